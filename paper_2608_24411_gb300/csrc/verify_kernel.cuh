// Fused verification kernel: one thread-block cluster walks one sequence's
// draft tree (Sec. 3, Algorithm 1, GetProxy).
//
// Data layout on chip.  The vocabulary is cut into C contiguous slices of L
// elements (L % 8 == 0), one per CTA of the cluster.  Each CTA keeps two fp32
// rows of its slice in shared memory:
//   W  the target row: raw logits -> exp((z - max) / T) -> the current
//      residual R, materialised after each rejection pass,
//   Q  the draft row:  raw logits -> exp((z - max) / T).
// bf16 rows land (bulk copy) in the upper half of W / Q and are widened in
// place.  A rejection never leaves the chip: its pass reads W and Q, writes
// the new residual back to W and produces the two sums the next residual
// needs; the cluster combines per-CTA sums through distributed shared
// memory.  The rows of a node are read from HBM exactly once.
//
// Lazy residual.  After rejection j the kernel knows only scalars
// (x0, Z, lambda, 1/norm) of the map R_j -> R_{j+1}; the next pass applies it
// element-wise while it computes the sums of rejection j+1.  The owner CTA of
// the next candidate publishes that candidate's stored values in the same
// exchange, so every CTA evaluates the next accept test from bit-identical
// operands without an extra round trip.
#pragma once
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "philox.cuh"
#include "ptx.cuh"

namespace rs {

constexpr int kErrTree = 1;
constexpr int kErrToken = 2;
constexpr int kErrNonfinite = 4;
constexpr int kErrEmpty = 8;
constexpr int kErrDepth = 16;
constexpr int kErrTimeout = 32;
constexpr int kInfoDegenerate = 256;

// Internal flag bits carried through the max exchange.
constexpr int kFlagTargetBad = 1;
constexpr int kFlagDraftBad = 2;
constexpr int kFlagTimeout = 4;

constexpr uint32_t kSpinLimit = 1u << 22;   // try_wait attempts before giving up
constexpr uint32_t kCopyChunk = 32768;      // bytes per bulk copy instruction
constexpr int kMaxCluster = 16;

struct VerifyParams {
  const void* zt;
  const void* zd;
  const int32_t* parents;
  const int32_t* cand;
  int32_t* out_tokens;
  int32_t* out_len;
  int32_t* out_nodes;
  float* out_dist;
  int32_t* out_rejects;
  int32_t* status;
  int64_t seq_stride;  // elements
  uint64_t seed;
  float scale_log2;    // log2(e) / T
  int32_t B, N, V, D;
  int32_t slice;       // L, elements per CTA
  int32_t npad;        // padded node count of the tree arrays
  int32_t mode;        // 0 ResiSpec, 1 SpecInfer
  int32_t use_tma;
};

struct __align__(16) Slot {
  float v[8];  // [0..3] reduced values, [4..5] published point values, [6] flags
  double d;    // sampler: this CTA's residual mass
  double pad;
};

struct __align__(16) Head {
  unsigned long long mbar[2];
  Slot slot[2];
  float red[32][8];
  float bc[8];
  double wsum[32];
  double cta_tot[kMaxCluster];
  int wcnt[32];
  int misc[4];
  double miscd[4];
};
constexpr int kHeadBytes = 2048;
static_assert(sizeof(Head) <= kHeadBytes, "head too large");

// ---------------------------------------------------------------- residual map
enum : int { kScale = 0, kIdent = 1, kResi = 2, kSpec = 3 };

struct Pending {
  int kind;
  int x0;     // rejected token (kResi)
  float a;    // scale (kScale) or 1 / norm (kResi, kSpec)
  float Z;    // budget (kResi)
  float lam;  // filled fraction of the capacity (kResi)
};

// R_{j+1}(x) from the stored R_j(x) = w and q(x) = qq.  Written with
// explicitly rounded intrinsics so that every caller computes the same bits.
template <int KIND>
__device__ __forceinline__ float apply_map(const Pending& P, float w, float qq, int idx) {
  if constexpr (KIND == kScale) {
    return __fmul_rn(w, P.a);
  } else if constexpr (KIND == kIdent) {
    return w;
  } else if constexpr (KIND == kResi) {
    // GetProxy: r = min(Z q, R) + lambda (R - min(Z q, R)) off x0, r(x0) = 0;
    // R' = r / sum r.
    if (idx == P.x0) return 0.f;
    const float m = fminf(__fmul_rn(P.Z, qq), w);
    return __fmul_rn(__fmaf_rn(P.lam, __fsub_rn(w, m), m), P.a);
  } else {
    // Eq. recur: R' = (R - q)_+ / sum.
    return __fmul_rn(fmaxf(__fsub_rn(w, qq), 0.f), P.a);
  }
}

__device__ __forceinline__ float apply_any(const Pending& P, float w, float qq, int idx) {
  switch (P.kind) {
    case kScale: return apply_map<kScale>(P, w, qq, idx);
    case kIdent: return apply_map<kIdent>(P, w, qq, idx);
    case kResi: return apply_map<kResi>(P, w, qq, idx);
    default: return apply_map<kSpec>(P, w, qq, idx);
  }
}

// ---------------------------------------------------------------- reductions
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// CTA reduction then cluster reduction through DSMEM.  v[0], v[1] are
// max-reduced when max01, otherwise summed; v[2..5] are summed; flags are
// OR-ed.  Butterfly reductions give bit-identical results in every lane and,
// because every CTA combines the same per-CTA partials in the same lanes, in
// every CTA of the cluster.
template <int NWARPS>
__device__ __forceinline__ void exchange(Head& H, const float (&v)[6], int flags, bool max01,
                                         int& par, uint32_t C, float (&out)[6], int& oflags) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float r[6];
#pragma unroll
  for (int k = 0; k < 6; ++k) r[k] = v[k];
  int f = flags;
#pragma unroll
  for (int o = 16; o; o >>= 1) {
#pragma unroll
    for (int k = 0; k < 6; ++k) {
      const float x = __shfl_xor_sync(0xffffffffu, r[k], o);
      r[k] = (max01 && k < 2) ? fmaxf(r[k], x) : r[k] + x;
    }
    f |= __shfl_xor_sync(0xffffffffu, f, o);
  }
  if (lane == 0) {
#pragma unroll
    for (int k = 0; k < 6; ++k) H.red[warp][k] = r[k];
    H.red[warp][6] = __int_as_float(f);
  }
  __syncthreads();
  if (warp == 0) {
#pragma unroll
    for (int k = 0; k < 6; ++k)
      r[k] = lane < NWARPS ? H.red[lane][k] : ((max01 && k < 2) ? -INFINITY : 0.f);
    f = lane < NWARPS ? __float_as_int(H.red[lane][6]) : 0;
#pragma unroll
    for (int o = 16; o; o >>= 1) {
#pragma unroll
      for (int k = 0; k < 6; ++k) {
        const float x = __shfl_xor_sync(0xffffffffu, r[k], o);
        r[k] = (max01 && k < 2) ? fmaxf(r[k], x) : r[k] + x;
      }
      f |= __shfl_xor_sync(0xffffffffu, f, o);
    }
    if (lane == 0) {
      Slot& s = H.slot[par];
#pragma unroll
      for (int k = 0; k < 6; ++k) s.v[k] = r[k];
      s.v[6] = __int_as_float(f);
      s.v[7] = 0.f;
    }
  }
  cluster_sync();
  if (warp == 0) {
    const float id01 = max01 ? -INFINITY : 0.f;
    float4 a = make_float4(id01, id01, 0.f, 0.f);
    float4 b = make_float4(0.f, 0.f, 0.f, 0.f);
    if (lane < (int)C) {
      const uint32_t addr = map_to_rank(smem_addr(&H.slot[par]), lane);
      a = ld_cluster_f4(addr);
      b = ld_cluster_f4(addr + 16);
    }
    r[0] = a.x; r[1] = a.y; r[2] = a.z; r[3] = a.w; r[4] = b.x; r[5] = b.y;
    f = lane < (int)C ? __float_as_int(b.z) : 0;
#pragma unroll
    for (int o = 16; o; o >>= 1) {
#pragma unroll
      for (int k = 0; k < 6; ++k) {
        const float x = __shfl_xor_sync(0xffffffffu, r[k], o);
        r[k] = (max01 && k < 2) ? fmaxf(r[k], x) : r[k] + x;
      }
      f |= __shfl_xor_sync(0xffffffffu, f, o);
    }
    if (lane == 0) {
#pragma unroll
      for (int k = 0; k < 6; ++k) H.bc[k] = r[k];
      H.bc[6] = __int_as_float(f);
    }
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < 6; ++k) out[k] = H.bc[k];
  oflags = __float_as_int(H.bc[6]);
  par ^= 1;
}

// ---------------------------------------------------------------- tree
// Children of `node` in ascending index order (children have larger
// indices than their parent) and their candidate tokens.  Uniform result.
template <int THREADS>
__device__ int gather_children(Head& H, const int16_t* par, int16_t* kids, int32_t* kidtok,
                               int node, int N, const int32_t* cand_b) {
  constexpr int NW = THREADS / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int count = 0;
  __syncthreads();
  for (int base = node + 1; base < N; base += THREADS) {
    const int c = base + (int)threadIdx.x;
    const bool f = c < N && par[c] == node;
    const unsigned m = __ballot_sync(0xffffffffu, f);
    if (lane == 0) H.wcnt[warp] = __popc(m);
    __syncthreads();
    int pre = 0, tot = 0;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const int x = H.wcnt[w];
      pre += w < warp ? x : 0;
      tot += x;
    }
    if (f) {
      const int pos = count + pre + __popc(m & ((1u << lane) - 1u));
      kids[pos] = (int16_t)c;
      kidtok[pos] = __ldg(cand_b + c);
    }
    count += tot;
    __syncthreads();
  }
  return count;
}

// ---------------------------------------------------------------- row I/O
// Starts the copies of this CTA's slice [lo, lo + nloc) of the target row
// (and of the draft row when need_draft) that begin at element row_base.
template <int THREADS, bool BF16>
__device__ __forceinline__ void issue_rows(Head& H, const VerifyParams& P, float* W, float* Q,
                                           size_t row_base, bool need_draft, int lo, int nloc) {
  const size_t row_off = row_base + (size_t)lo;
  const int L = P.slice;
  // Earlier generic accesses to W / Q must be ordered before the copies.
  fence_proxy_async_smem();
  __syncthreads();
  constexpr uint32_t es = BF16 ? 2u : 4u;
  if (P.use_tma) {
    if (threadIdx.x == 0) {
      const uint32_t bytes = (uint32_t)nloc * es;
      const uint32_t dst_off = BF16 ? 2u * (uint32_t)L : 0u;
      for (int which = 0; which < (need_draft ? 2 : 1); ++which) {
        const uint32_t bar = smem_addr(&H.mbar[which]);
        const char* src = static_cast<const char*>(which ? P.zd : P.zt) + row_off * es;
        const uint32_t dst = smem_addr(which ? Q : W) + dst_off;
        mbar_arrive_expect_tx(bar, bytes);
        for (uint32_t o = 0; o < bytes; o += kCopyChunk)
          bulk_g2s(dst + o, src + o, min(kCopyChunk, bytes - o), bar);
      }
    }
  } else {
    for (int which = 0; which < (need_draft ? 2 : 1); ++which) {
      float* dst = which ? Q : W;
      if constexpr (BF16) {
        const uint16_t* src = static_cast<const uint16_t*>(which ? P.zd : P.zt) + row_off;
        uint16_t* raw = reinterpret_cast<uint16_t*>(dst) + L;
        for (int i = threadIdx.x; i < nloc; i += THREADS) raw[i] = __ldg(src + i);
      } else {
        const float* src = static_cast<const float*>(which ? P.zd : P.zt) + row_off;
        for (int i = threadIdx.x; i < nloc; i += THREADS) dst[i] = __ldg(src + i);
      }
    }
  }
}

__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity) {
  for (uint32_t it = 0; it < kSpinLimit; ++it)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

__device__ __forceinline__ bool bad_logit(float x) { return isnan(x) || x == INFINITY; }

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Max over the valid part of the slice of both raw rows, with the
// non-finite check of the error contract.
template <int THREADS, bool BF16>
__device__ __forceinline__ void max_pass(const float* W, const float* Q, int L, int nloc,
                                         bool need_draft, float& mt, float& md, int& flags) {
  mt = -INFINITY;
  md = -INFINITY;
  for (int which = 0; which < (need_draft ? 2 : 1); ++which) {
    const float* buf = which ? Q : W;
    float m = -INFINITY;
    bool bad = false;
    if constexpr (BF16) {
      const uint16_t* raw = reinterpret_cast<const uint16_t*>(buf) + L;
      for (int i = threadIdx.x * 8; i < nloc; i += THREADS * 8) {
        const uint4 r = *reinterpret_cast<const uint4*>(raw + i);
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float a = bf16_lo(w[k]), b = bf16_hi(w[k]);
          if (i + 2 * k < nloc) { bad |= bad_logit(a); m = fmaxf(m, a); }
          if (i + 2 * k + 1 < nloc) { bad |= bad_logit(b); m = fmaxf(m, b); }
        }
      }
    } else {
      for (int i = threadIdx.x * 4; i < nloc; i += THREADS * 4) {
        const float4 r = *reinterpret_cast<const float4*>(buf + i);
        const float x[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int k = 0; k < 4; ++k)
          if (i + k < nloc) { bad |= bad_logit(x[k]); m = fmaxf(m, x[k]); }
      }
    }
    if (which) { md = m; flags |= bad ? kFlagDraftBad : 0; }
    else { mt = m; flags |= bad ? kFlagTargetBad : 0; }
  }
}

// e = exp((z - M) / T) over the slice (0 beyond the valid part), sums, and
// the stored values of token `x1` when this CTA owns it.
template <int THREADS, bool BF16>
__device__ __forceinline__ void exp_pass(float* W, float* Q, int L, int nloc, int lo,
                                         bool need_draft, float Mt, float Md, float c,
                                         int x1, float& st, float& sd, float& pubW,
                                         float& pubQ) {
  st = 0.f;
  sd = 0.f;
  pubW = 0.f;
  pubQ = 0.f;
  if constexpr (BF16) {
    constexpr int CH = THREADS * 8;
    for (int base = 0; base < L; base += CH) {
      const int i = base + (int)threadIdx.x * 8;
      float et[8], ed[8];
#pragma unroll
      for (int which = 0; which < 2; ++which) {
        float* e = which ? ed : et;
#pragma unroll
        for (int k = 0; k < 8; ++k) e[k] = 0.f;
        if (which == 1 && !need_draft) continue;
        if (i < nloc) {
          const uint16_t* raw = reinterpret_cast<const uint16_t*>(which ? Q : W) + L;
          const uint4 r = *reinterpret_cast<const uint4*>(raw + i);
          const uint32_t w[4] = {r.x, r.y, r.z, r.w};
          const float M = which ? Md : Mt;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            if (i + 2 * k < nloc) e[2 * k] = exp2f(__fmul_rn(__fsub_rn(bf16_lo(w[k]), M), c));
            if (i + 2 * k + 1 < nloc)
              e[2 * k + 1] = exp2f(__fmul_rn(__fsub_rn(bf16_hi(w[k]), M), c));
          }
        }
      }
      __syncthreads();  // every raw value of this chunk has been read
      if (i < L) {
        float4* wt = reinterpret_cast<float4*>(W + i);
        wt[0] = make_float4(et[0], et[1], et[2], et[3]);
        wt[1] = make_float4(et[4], et[5], et[6], et[7]);
        if (need_draft) {
          float4* wd = reinterpret_cast<float4*>(Q + i);
          wd[0] = make_float4(ed[0], ed[1], ed[2], ed[3]);
          wd[1] = make_float4(ed[4], ed[5], ed[6], ed[7]);
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          st += et[k];
          sd += ed[k];
          if (lo + i + k == x1) { pubW = et[k]; pubQ = ed[k]; }
        }
      }
    }
  } else {
    for (int i = threadIdx.x * 4; i < L; i += THREADS * 4) {
      for (int which = 0; which < (need_draft ? 2 : 1); ++which) {
        float* buf = which ? Q : W;
        const float M = which ? Md : Mt;
        float4 r = *reinterpret_cast<float4*>(buf + i);
        float x[4] = {r.x, r.y, r.z, r.w};
        float s = 0.f;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          x[k] = (i + k < nloc) ? exp2f(__fmul_rn(__fsub_rn(x[k], M), c)) : 0.f;
          s += x[k];
          if (lo + i + k == x1) { if (which) pubQ = x[k]; else pubW = x[k]; }
        }
        *reinterpret_cast<float4*>(buf + i) = make_float4(x[0], x[1], x[2], x[3]);
        if (which) sd += s; else st += s;
      }
    }
  }
}

// One rejection pass: materialise R_j = map(W) into W and accumulate the
// sums of rejection j (ResiSpec: sum min(Z q, R) and sum (R - min(Z q, R))
// over x != x0; SpecInfer: sum (R - q)_+), publishing the next candidate.
template <int THREADS, int KIND, bool RESI>
__device__ __forceinline__ void reject_pass(float* W, const float* Q, int L, int lo,
                                            const Pending& P, float invSd, int x0, float Z,
                                            int xn, float& s1, float& s2, float& pubW,
                                            float& pubQ) {
  s1 = 0.f;
  s2 = 0.f;
  pubW = 0.f;
  pubQ = 0.f;
  for (int i = threadIdx.x * 4; i < L; i += THREADS * 4) {
    float4 wv = *reinterpret_cast<float4*>(W + i);
    const float4 qv = *reinterpret_cast<const float4*>(Q + i);
    float w[4] = {wv.x, wv.y, wv.z, wv.w};
    const float qr[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int idx = lo + i + k;
      const float qq = __fmul_rn(qr[k], invSd);
      const float R = apply_map<KIND>(P, w[k], qq, idx);
      w[k] = R;
      if constexpr (RESI) {
        if (idx != x0) {
          const float m = fminf(__fmul_rn(Z, qq), R);
          s1 += m;
          s2 += __fsub_rn(R, m);
        }
      } else {
        s1 += fmaxf(__fsub_rn(R, qq), 0.f);
      }
      if (idx == xn) { pubW = R; pubQ = qr[k]; }
    }
    *reinterpret_cast<float4*>(W + i) = make_float4(w[0], w[1], w[2], w[3]);
  }
}

template <int THREADS, bool RESI>
__device__ __forceinline__ void reject_pass_any(float* W, const float* Q, int L, int lo,
                                                const Pending& P, float invSd, int x0, float Z,
                                                int xn, float& s1, float& s2, float& pubW,
                                                float& pubQ) {
  switch (P.kind) {
    case kScale:
      reject_pass<THREADS, kScale, RESI>(W, Q, L, lo, P, invSd, x0, Z, xn, s1, s2, pubW, pubQ);
      break;
    case kIdent:
      reject_pass<THREADS, kIdent, RESI>(W, Q, L, lo, P, invSd, x0, Z, xn, s1, s2, pubW, pubQ);
      break;
    case kResi:
      reject_pass<THREADS, kResi, RESI>(W, Q, L, lo, P, invSd, x0, Z, xn, s1, s2, pubW, pubQ);
      break;
    default:
      reject_pass<THREADS, kSpec, RESI>(W, Q, L, lo, P, invSd, x0, Z, xn, s1, s2, pubW, pubQ);
      break;
  }
}

// ---------------------------------------------------------------- sampler
// Inverse-CDF draw: the smallest token x with C(x) > u * C(V-1), found
// hierarchically (CTA slice, then warp range, then 32-token group, then
// lane).  Groups of 32 are summed in fp32; the running sums above them are
// kept in fp64 (a few dozen additions per CTA) so that the prefix rounding
// stays far below the near-tie margin.  Each level falls back to its last
// unit with positive mass, so the result always has R(x) > 0.  Returns
// false when the residual has no mass.
template <int THREADS>
__device__ bool sample_final(Head& H, const VerifyParams& P, const float* W, const float* Q,
                             const Pending& Pm, float invSd, int b, int row, int depth,
                             int lo, int nloc, uint32_t rank, uint32_t C, int& par) {
  constexpr int NW = THREADS / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int L = P.slice;
  const int Lw = ((L + NW * 32 - 1) / (NW * 32)) * 32;
  const int wb = warp * Lw;
  const int we = min(wb + Lw, nloc);
  float* dist = P.out_dist ? P.out_dist + (size_t)b * P.V + lo : nullptr;
  double acc = 0.0;
  for (int g = wb; g < we; g += 32) {
    const int i = g + lane;
    float v = 0.f;
    if (i < we) {
      v = apply_any(Pm, W[i], __fmul_rn(Q[i], invSd), lo + i);
      if (dist) dist[i] = v;
    }
    acc += (double)warp_sum(v);
  }
  if (lane == 0) H.wsum[warp] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < NW; ++w) t += H.wsum[w];
    H.slot[par].d = t;
  }
  cluster_sync();
  if (warp == 0) {
    if (lane < (int)C) {
      const uint32_t addr = map_to_rank(smem_addr(&H.slot[par].d), lane);
      H.cta_tot[lane] = ld_cluster_f64(addr);
    }
    __syncwarp();
    if (lane == 0) {
      const double u = (double)uniform_draw(P.seed, (uint32_t)b, (uint32_t)row, 1);
      double total = 0.0;
      for (uint32_t r = 0; r < C; ++r) total += H.cta_tot[r];
      int cstar = -1, force = 0;
      double before = 0.0;
      if (total > 0.0) {
        const double tau = u * total;
        double a = 0.0, last_before = 0.0;
        int last = -1;
        for (uint32_t r = 0; r < C; ++r) {
          const double nx = a + H.cta_tot[r];
          if (H.cta_tot[r] > 0.0) { last = (int)r; last_before = a; }
          if (nx > tau) { cstar = (int)r; before = a; break; }
          a = nx;
        }
        if (cstar < 0) { cstar = last; before = last_before; force = 1; }
        H.miscd[0] = tau - before;
      }
      H.misc[0] = cstar;
      H.misc[1] = force;
    }
  }
  __syncthreads();
  par ^= 1;
  const int cstar = H.misc[0];
  if (cstar < 0) return false;
  if ((int)rank != cstar) return true;
  // This CTA holds the draw: find the warp range, then the group, then the lane.
  if (threadIdx.x == 0) {
    const double t = H.miscd[0];
    int force = H.misc[1];
    double a = 0.0, last_before = 0.0;
    int wstar = -1, last = -1;
    for (int w = 0; w < NW; ++w) {
      const double s = H.wsum[w];
      if (s > 0.0) { last = w; last_before = a; }
      if (!force && a + s > t) { wstar = w; break; }
      a += s;
    }
    if (wstar < 0) { wstar = last; a = last_before; force = 1; }
    H.misc[2] = wstar;
    H.misc[3] = force;
    H.miscd[1] = t - a;
  }
  __syncthreads();
  if (warp == H.misc[2]) {
    const double t = H.miscd[1];
    bool force = H.misc[3] != 0;
    double a = 0.0, last_before = 0.0;
    int gstar = -1, last = -1;
    for (int g = wb; g < we; g += 32) {
      const int i = g + lane;
      const float v = i < we ? apply_any(Pm, W[i], __fmul_rn(Q[i], invSd), lo + i) : 0.f;
      const double s = (double)warp_sum(v);
      if (s > 0.0) { last = g; last_before = a; }
      if (!force && a + s > t) { gstar = g; break; }
      a += s;
    }
    if (gstar < 0) { gstar = last; a = last_before; force = true; }
    const int i = gstar + lane;
    const float v = i < we ? apply_any(Pm, W[i], __fmul_rn(Q[i], invSd), lo + i) : 0.f;
    double s = (double)v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const double n = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += n;
    }
    const double tl = t - a;
    const unsigned cross = __ballot_sync(0xffffffffu, !force && s > tl);
    const unsigned pos = __ballot_sync(0xffffffffu, v > 0.f);
    const int l = cross ? __ffs(cross) - 1 : 31 - __clz(pos);
    if (lane == 0) P.out_tokens[(size_t)b * (P.D + 1) + depth] = lo + gstar + l;
  }
  return true;
}

// ---------------------------------------------------------------- kernel
template <int THREADS, bool BF16>
__global__ void __launch_bounds__(THREADS, 1) verify_kernel(const VerifyParams P) {
  constexpr int NW = THREADS / 32;
  extern __shared__ __align__(128) unsigned char smem[];
  Head& H = *reinterpret_cast<Head*>(smem);
  const int L = P.slice;
  float* W = reinterpret_cast<float*>(smem + kHeadBytes);
  float* Q = W + L;
  int16_t* par = reinterpret_cast<int16_t*>(Q + L);
  int16_t* kids = par + P.npad;
  int32_t* kidtok = reinterpret_cast<int32_t*>(kids + P.npad);
  uint8_t* haschild = reinterpret_cast<uint8_t*>(kidtok + P.npad);

  const int tid = threadIdx.x;
  const uint32_t rank = cluster_ctarank();
  const uint32_t C = cluster_nctarank();
  const int b = (int)cluster_id_x();
  const int N = P.N, V = P.V, D = P.D;
  const int lo = (int)rank * L;
  const int nloc = max(0, min(V, lo + L) - lo);
  const int32_t* cand_b = P.cand + (size_t)b * N;

  if (tid == 0) {
    mbar_init(smem_addr(&H.mbar[0]), 1);
    mbar_init(smem_addr(&H.mbar[1]), 1);
    fence_mbar_init();
  }
  for (int i = tid; i <= N; i += THREADS) haschild[i] = 0;
  __syncthreads();
  int bad = 0;
  for (int c = tid; c < N; c += THREADS) {
    const int p = __ldg(P.parents + c);
    const bool ok = p >= -1 && p < c;
    bad |= !ok;
    par[c] = (int16_t)(ok ? p : -2);
    if (ok) haschild[p + 1] = 1;
  }
  const bool tree_bad = __syncthreads_or(bad) != 0;

  int err = tree_bad ? kErrTree : 0;
  int info = 0;
  int depth = 0, rejects = 0;
  int node = -1, row = 0;
  uint32_t ph0 = 0, ph1 = 0;
  int rpar = 0;
  bool timed_out = false;
  const float c = P.scale_log2;

  if (!err)
    issue_rows<THREADS, BF16>(H, P, W, Q, (size_t)b * P.seq_stride, haschild[0] != 0, lo, nloc);

  while (!err) {
    const bool need_draft = haschild[node + 1] != 0;
    const int nk = need_draft ? gather_children<THREADS>(H, par, kids, kidtok, node, N, cand_b) : 0;

    // ---- rows of this node: wait for the copies
    if (P.use_tma) {
      bool ok = wait_bar(smem_addr(&H.mbar[0]), ph0);
      ph0 ^= 1;
      if (need_draft) {
        ok = wait_bar(smem_addr(&H.mbar[1]), ph1) && ok;
        ph1 ^= 1;
      }
      timed_out |= !ok;
    } else {
      __syncthreads();
    }

    // ---- tempered normaliser: max, then exp and sums (S2)
    float mt, md;
    int flags = timed_out ? kFlagTimeout : 0;
    if (!timed_out) max_pass<THREADS, BF16>(W, Q, L, nloc, need_draft, mt, md, flags);
    else { mt = 0.f; md = 0.f; }
    float v[6] = {mt, md, 0.f, 0.f, 0.f, 0.f}, o[6];
    int oflags;
    exchange<NW>(H, v, flags, true, rpar, C, o, oflags);
    const float Mt = o[0], Md = o[1];
    if (oflags & kFlagTimeout) { err |= kErrTimeout; break; }
    if (oflags & kFlagTargetBad) { err |= kErrNonfinite; break; }
    if (Mt == -INFINITY) { err |= kErrEmpty; break; }
    if (need_draft && (oflags & kFlagDraftBad)) { err |= kErrNonfinite; break; }
    if (need_draft && Md == -INFINITY) { err |= kErrEmpty; break; }

    const int x1 = nk > 0 ? kidtok[0] : -1;
    float st, sd, pw, pq;
    exp_pass<THREADS, BF16>(W, Q, L, nloc, lo, need_draft, Mt, Md, c, x1, st, sd, pw, pq);
    float v2[6] = {st, sd, 0.f, 0.f, pw, pq};
    exchange<NW>(H, v2, 0, false, rpar, C, o, oflags);
    const float invSt = __frcp_rn(o[0]);
    const float invSd = need_draft ? __frcp_rn(o[1]) : 0.f;
    float pubW = o[4], pubQ = o[5];
    Pending Pm{kScale, -1, invSt, 0.f, 0.f};

    if (!need_draft) {
      // accepted leaf (or a root without children): bonus token from p
      if (!sample_final<THREADS>(H, P, W, Q, Pm, invSd, b, row, depth, lo, nloc, rank, C, rpar))
        err |= kErrEmpty;
      break;
    }

    // ---- sequential accept tests over the children (S3), shaping on reject
    int accepted = -1, acc_tok = -1;
    for (int j = 0; j < nk; ++j) {
      const int cnode = kids[j];
      const int x = kidtok[j];
      if (x < 0 || x >= V) { err |= kErrToken; break; }
      const float qx = __fmul_rn(pubQ, invSd);
      const float Rx = apply_any(Pm, pubW, qx, x);
      const float u = uniform_draw(P.seed, (uint32_t)b, (uint32_t)(cnode + 1), 0);
      if (__fmul_rn(u, qx) < Rx) { accepted = cnode; acc_tok = x; break; }
      rejects += 1;
      const int xn = j + 1 < nk ? kidtok[j + 1] : -1;
      float s1 = 0.f, s2 = 0.f, pw2 = 0.f, pq2 = 0.f;
      if (P.mode == 0) {
        const float Z = __fsub_rn(qx, Rx);
        if (!(Z > 0.f)) {
          // degenerate rejection: keep R, fetch the next candidate's values
          info |= kInfoDegenerate;
          if (tid == 0 && xn >= lo && xn < lo + nloc) { pw2 = W[xn - lo]; pq2 = Q[xn - lo]; }
          float v3[6] = {0.f, 0.f, 0.f, 0.f, pw2, pq2};
          exchange<NW>(H, v3, 0, false, rpar, C, o, oflags);
          pubW = o[4];
          pubQ = o[5];
          continue;
        }
        reject_pass_any<THREADS, true>(W, Q, L, lo, Pm, invSd, x, Z, xn, s1, s2, pw2, pq2);
        float v3[6] = {s1, s2, 0.f, 0.f, pw2, pq2};
        exchange<NW>(H, v3, 0, false, rpar, C, o, oflags);
        const float S1 = o[0], S2 = o[1];
        const float delta = __fsub_rn(Z, S1);
        const float lam = S2 > 0.f ? fminf(fmaxf(__fdiv_rn(delta, S2), 0.f), 1.f) : 0.f;
        const float norm = __fmaf_rn(lam, S2, S1);
        if (norm > 0.f) Pm = Pending{kResi, x, __frcp_rn(norm), Z, lam};
        else { Pm = Pending{kIdent, -1, 1.f, 0.f, 0.f}; info |= kInfoDegenerate; }
      } else {
        reject_pass_any<THREADS, false>(W, Q, L, lo, Pm, invSd, x, 0.f, xn, s1, s2, pw2, pq2);
        float v3[6] = {s1, 0.f, 0.f, 0.f, pw2, pq2};
        exchange<NW>(H, v3, 0, false, rpar, C, o, oflags);
        if (o[0] > 0.f) Pm = Pending{kSpec, -1, __frcp_rn(o[0]), 0.f, 0.f};
        else { Pm = Pending{kIdent, -1, 1.f, 0.f, 0.f}; info |= kInfoDegenerate; }
      }
      pubW = o[4];
      pubQ = o[5];
    }
    if (err) break;

    if (accepted < 0) {
      // every child rejected: residual draw (Algorithm 1, last step)
      if (!sample_final<THREADS>(H, P, W, Q, Pm, invSd, b, row, depth, lo, nloc, rank, C, rpar))
        err |= kErrEmpty;
      break;
    }
    if (depth >= D) { err |= kErrDepth; break; }
    if (rank == 0 && tid == 0) {
      P.out_tokens[(size_t)b * (D + 1) + depth] = acc_tok;
      if (P.out_nodes) P.out_nodes[(size_t)b * D + depth] = accepted;
    }
    depth += 1;
    node = accepted;
    row = accepted + 1;
    issue_rows<THREADS, BF16>(H, P, W, Q, (size_t)b * P.seq_stride + (size_t)row * V,
                              haschild[node + 1] != 0, lo, nloc);
  }

  if (rank == 0 && tid == 0) {
    int32_t* toks = P.out_tokens + (size_t)b * (D + 1);
    if (err) {
      for (int i = 0; i <= D; ++i) toks[i] = -1;
      if (P.out_nodes)
        for (int i = 0; i < D; ++i) P.out_nodes[(size_t)b * D + i] = -1;
      P.out_len[b] = -1;
    } else {
      for (int i = depth + 1; i <= D; ++i) toks[i] = -1;
      if (P.out_nodes)
        for (int i = depth; i < D; ++i) P.out_nodes[(size_t)b * D + i] = -1;
      P.out_len[b] = depth;
    }
    if (P.out_rejects) P.out_rejects[b] = rejects;
    if (P.status && (err | info)) atomicOr(P.status, err | info);
  }
  if (timed_out && P.use_tma && tid == 0) {
    // give outstanding copies a bounded chance to land before the CTA exits
    wait_bar(smem_addr(&H.mbar[0]), ph0 ^ 1);
    wait_bar(smem_addr(&H.mbar[1]), ph1 ^ 1);
  }
  cluster_sync();  // no CTA leaves while a peer may still read its slots
}

// Device Philox draws for tests.
__global__ void uniforms_kernel(uint64_t seed, const int32_t* seq, const int32_t* row, int n,
                                float* u0, float* u1) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const U64x4 r = philox4x64_10((uint64_t)(uint32_t)row[i], (uint64_t)(uint32_t)seq[i], 0, 0,
                                seed, 0);
  u0[i] = u24(r.w[0]);
  u1[i] = u24(r.w[1]);
}

}  // namespace rs
