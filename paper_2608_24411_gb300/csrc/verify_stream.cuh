// Streaming verification kernel: one thread-block cluster walks one
// sequence's draft tree (Sec. 3, Algorithm 1, GetProxy), like the resident
// kernel in verify_kernel.cuh, but keeps no logit row on chip.
//
// Why.  Holding both fp32 rows of a sequence in shared memory costs
// 8 bytes per vocabulary entry, so at V = 151936 only about 28 sequences fit
// in the GPU's 34.6 MB of shared memory, and at V = 256000 about 16: the HBM
// then idles while those few sequences run their serial accept/reject
// chains.  Here the on-chip state of a sequence is a few kilobytes of
// scalars, so every sequence of a large batch is in flight at once and the
// rows of all of them (64 x 1.2 MB at V = 151936) stay in the 126 MB L2
// between the passes of a visit.  Rows are read from HBM once per visit.
//
// Passes.  Each CTA owns the slice [lo, lo + nloc) of the vocabulary and
// streams it through a ring of S shared-memory stages, one chunk (2 THREADS
// 16-byte vectors per row) per stage, filled by 1-D bulk copies (TMA) that
// complete on one mbarrier per stage.  A visit runs
//   NORM   online (reference, sum) of 2^(z c) per thread, c = log2(e) / T,
//          then one cluster exchange gives the global (M, S) of each row;
//   REJ    once per rejected candidate (Algorithm 1, GetProxy / Eq. recur):
//          recomputes p = 2^(z_t c - M_t) / S_t and q likewise from the raw
//          logits (L2 hits), applies the residual maps of the earlier
//          rejections in order, and sums the terms of the new map;
//   SAMP   residual or bonus draw, in the CTA that holds the threshold.
// After the normaliser every value is a function of the raw logit and
// cluster-wide scalars only, so any thread may compute any element and every
// CTA evaluates the accept tests itself from the candidates' raw logits.
#pragma once
#include "verify_kernel.cuh"

namespace rs {

constexpr int kMaxStages = 4;
constexpr int kMaxMaps = 128;          // residual maps per node (rejections with a map)
constexpr int kMaxKids = kMaxMaps;      // children per node the streaming kernel walks
constexpr int kErrFanout = 64;

struct __align__(16) StreamHead {
  unsigned long long fbar[kMaxStages];  // stage full barriers
  float mZ[kMaxMaps];                   // ResiSpec budget Z of map i
  float mlam[kMaxMaps];                 // ResiSpec filled fraction lambda of map i
  float ma[kMaxMaps];                   // 1 / normaliser of map i
  int rej[kMaxMaps];                    // tokens whose residual is 0 (ResiSpec maps)
  float kzt[kMaxKids];                  // raw target / draft logits of the children's tokens
  float kzd[kMaxKids];
  int knode[kMaxKids];                  // the children, ascending
  int nkids;
  int nmaps;
  int fz[4];
};
constexpr int kStreamHeadBytes = 4096;
static_assert(sizeof(StreamHead) <= kStreamHeadBytes, "stream head too large");

template <int THREADS, bool BF16>
struct StreamGeom {
  static constexpr int VEC = BF16 ? 8 : 4;            // elements per 16-byte vector
  static constexpr int VPT = 2;                       // vectors per thread per chunk and row
  static constexpr int CV = VPT * THREADS;            // vectors per chunk and row
  static constexpr int CE = CV * VEC;                 // elements per chunk and row
  static constexpr uint32_t RB = (uint32_t)CV * 16u;  // bytes per chunk and row
  static constexpr uint32_t SB = 2u * RB;             // bytes per stage (target, draft)
};

// Ring bookkeeping; every thread holds identical copies.
struct Ring {
  unsigned char* buf;  // S stages of SB bytes
  uint32_t addr;       // shared address of buf
  uint32_t bar0;       // shared address of fbar[0]
  int S;
  uint32_t issued;     // chunks issued so far
  uint32_t consumed;   // chunks consumed so far
  bool tma;
  bool ok;             // false once a stage wait timed out
};

// Raw logits of vector g of a stage row; elements at or beyond `valid` read
// as -inf (the ragged end of a slice in the plain-load path).
template <bool BF16>
__device__ __forceinline__ void load_vec(const unsigned char* row, int g, int valid,
                                         float (&z)[BF16 ? 8 : 4]) {
  if constexpr (BF16) {
    const uint4 r = reinterpret_cast<const uint4*>(row)[g];
    const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      z[2 * j] = bf16_lo(w[j]);
      z[2 * j + 1] = bf16_hi(w[j]);
    }
  } else {
    const float4 r = reinterpret_cast<const float4*>(row)[g];
    z[0] = r.x; z[1] = r.y; z[2] = r.z; z[3] = r.w;
  }
  constexpr int VEC = BF16 ? 8 : 4;
  if (valid < VEC) {
#pragma unroll
    for (int j = 0; j < VEC; ++j)
      if (j >= valid) z[j] = -INFINITY;
  }
}

__device__ __forceinline__ float raw_logit(const void* base, size_t i, bool bf16) {
  if (bf16) {
    const uint16_t h = __ldg(static_cast<const uint16_t*>(base) + i);
    return __uint_as_float((uint32_t)h << 16);
  }
  return __ldg(static_cast<const float*>(base) + i);
}

// Streams this CTA's slice of `rows` rows (1: target; 2: target and draft,
// each starting at element `off` of its tensor) through the ring, calling
// body(target_stage_row, draft_stage_row, k, clen) for chunk k of clen
// elements with all threads.  body returns true (uniformly) to end the pass
// after its chunk; copies already in flight are then waited for (bounded).
// pre() runs once with all threads after the first copies are issued.
template <int THREADS, bool BF16, class Pre, class Body>
__device__ __forceinline__ void stream_pass_pre(Ring& R, const VerifyParams& P, int rows,
                                                size_t off, int nloc, Pre&& pre, Body&& body) {
  using G = StreamGeom<THREADS, BF16>;
  constexpr uint32_t es = BF16 ? 2u : 4u;
  const int NK = (nloc + G::CE - 1) / G::CE;
  const char* st = static_cast<const char*>(P.zt) + off * es;
  const char* sd = static_cast<const char*>(P.zd) + off * es;
  auto issue = [&](int k) {
    const uint32_t slot = R.issued % (uint32_t)R.S;
    if (threadIdx.x == 0) {
      const uint32_t bytes = (uint32_t)min(G::CE, nloc - k * G::CE) * es;
      const uint32_t bar = R.bar0 + 8u * slot;
      const uint32_t dst = R.addr + slot * G::SB;
      fence_proxy_async_smem();  // earlier generic accesses to the stage come first
      mbar_arrive_expect_tx(bar, (uint32_t)rows * bytes);
      bulk_g2s(dst, st + (size_t)k * G::CE * es, bytes, bar);
      if (rows == 2) bulk_g2s(dst + G::RB, sd + (size_t)k * G::CE * es, bytes, bar);
    }
    R.issued += 1;
  };
  if (R.tma)
    for (int k = 0; k < min(R.S, NK); ++k) issue(k);
  pre();
  for (int k = 0; k < NK; ++k) {
    const uint32_t slot = R.consumed % (uint32_t)R.S;
    unsigned char* s0 = R.buf + slot * G::SB;
    const int clen = min(G::CE, nloc - k * G::CE);
    if (R.tma) {
      // after one timed-out wait the pass runs on without waiting (the
      // sequence reports ERR_TIMEOUT)
      if (R.ok) R.ok = wait_bar(R.bar0 + 8u * slot, (R.consumed / (uint32_t)R.S) & 1u);
    } else {
      for (int w = 0; w < rows; ++w) {
        if constexpr (BF16) {
          const uint16_t* src = reinterpret_cast<const uint16_t*>(w ? sd : st) + (size_t)k * G::CE;
          uint16_t* dst = reinterpret_cast<uint16_t*>(s0 + w * G::RB);
          for (int i = threadIdx.x; i < clen; i += THREADS) dst[i] = __ldg(src + i);
        } else {
          const float* src = reinterpret_cast<const float*>(w ? sd : st) + (size_t)k * G::CE;
          float* dst = reinterpret_cast<float*>(s0 + w * G::RB);
          for (int i = threadIdx.x; i < clen; i += THREADS) dst[i] = __ldg(src + i);
        }
      }
      __syncthreads();
    }
    const bool stop = body(s0, s0 + G::RB, k, clen);
    R.consumed += 1;
    __syncthreads();  // every thread is done with the stage
    if (stop) break;
    if (R.tma && k + R.S < NK) issue(k + R.S);
  }
  while (R.consumed < R.issued) {  // copies of an ended pass still land
    const uint32_t slot = R.consumed % (uint32_t)R.S;
    if (R.ok) R.ok = wait_bar(R.bar0 + 8u * slot, (R.consumed / (uint32_t)R.S) & 1u);
    R.consumed += 1;
  }
}

template <int THREADS, bool BF16, class Body>
__device__ __forceinline__ void stream_pass(Ring& R, const VerifyParams& P, int rows, size_t off,
                                            int nloc, Body&& body) {
  stream_pass_pre<THREADS, BF16>(R, P, rows, off, nloc, [] {}, body);
}

// Online (reference, sum) of 2^(z c) over one thread's values of a chunk:
// the reference m (log2 units) is raised when a value exceeds it by more
// than 64 binary orders, and the sum is rescaled.  NaN or +inf makes the
// sum non-finite (detected by the caller).
template <int N>
__device__ __forceinline__ void norm_accumulate(const float (&z)[N], float c, float& m,
                                                float& s) {
  float vmax = -INFINITY;
#pragma unroll
  for (int j = 0; j < N; ++j) vmax = fmaxf(vmax, z[j]);
  if (__fmaf_rn(vmax, c, -m) > kRebaseLog2) {
    const float mnew = __fmul_rn(vmax, c);
    if (m != -INFINITY) s = __fmul_rn(s, ex2(__fsub_rn(m, mnew)));
    m = mnew;
  }
  if (m == -INFINITY) {  // nothing finite seen yet: every value is -inf or NaN
#pragma unroll
    for (int j = 0; j < N; ++j)
      if (isnan(z[j])) s = __int_as_float(0x7fc00000);
  } else {
    float t = 0.f;
#pragma unroll
    for (int j = 0; j < N; ++j) t += ex2(__fmaf_rn(z[j], c, -m));
    s += t;
  }
}

// Cluster-wide scalars of a visit after the normaliser.
struct VisitScalars {
  float c;           // log2(e) / T
  float Mt, invSt;   // target: global reference, 1 / sum
  float Md, invSd;   // draft
};

// p and q of one element from its raw logits.
__device__ __forceinline__ float prob_of(float z, float c, float M, float inv) {
  return __fmul_rn(ex2(__fmaf_rn(z, c, -M)), inv);
}

// The residual after the first nm maps, element-wise (no rejected-token
// zeroing: the caller applies it).  ResiSpec map: GetProxy residual
// r = min(Z q, R) + lambda (R - min(Z q, R)), R' = r / sum r; SpecInfer map:
// R' = (R - q)_+ / sum (Eq. recur).
template <bool RESI>
__device__ __forceinline__ float apply_chain(const StreamHead& S2, int nm, float R, float q) {
  for (int i = 0; i < nm; ++i) {
    if constexpr (RESI) {
      const float m = fminf(__fmul_rn(S2.mZ[i], q), R);
      R = __fmul_rn(__fmaf_rn(S2.mlam[i], __fsub_rn(R, m), m), S2.ma[i]);
    } else {
      R = __fmul_rn(fmaxf(__fsub_rn(R, q), 0.f), S2.ma[i]);
    }
  }
  return R;
}

template <int VEC, bool RESI>
__device__ __forceinline__ void apply_chain_vec(const StreamHead& S2, int nm, float (&R)[VEC],
                                                const float (&q)[VEC]) {
  for (int i = 0; i < nm; ++i) {
    if constexpr (RESI) {
      const float Z = S2.mZ[i], lam = S2.mlam[i], a = S2.ma[i];
#pragma unroll
      for (int j = 0; j < VEC; ++j) {
        const float m = fminf(__fmul_rn(Z, q[j]), R[j]);
        R[j] = __fmul_rn(__fmaf_rn(lam, __fsub_rn(R[j], m), m), a);
      }
    } else {
      const float a = S2.ma[i];
#pragma unroll
      for (int j = 0; j < VEC; ++j) R[j] = __fmul_rn(fmaxf(__fsub_rn(R[j], q[j]), 0.f), a);
    }
  }
}

// Zero the residual at rejected tokens (ResiSpec: r(x0) = 0 and the later
// maps keep a zero at zero) inside the vector starting at token `base`.
template <int VEC>
__device__ __forceinline__ void zero_rejected(const StreamHead& S2, int nm, int base,
                                              float (&R)[VEC]) {
  for (int i = 0; i < nm; ++i) {
    const unsigned d = (unsigned)(S2.rej[i] - base);
    if (d < (unsigned)VEC) {
#pragma unroll
      for (int j = 0; j < VEC; ++j)
        if ((unsigned)j == d) R[j] = 0.f;
    }
  }
}

// Final value (the distribution being sampled) of the VEC elements of a
// vector: p when no map is pending, else the residual.
template <int VEC>
__device__ __forceinline__ void final_values(const StreamHead& S2, const VisitScalars& K,
                                             bool resi, int nm, int base, const float (&zt)[VEC],
                                             const float (&zd)[VEC], float (&v)[VEC]) {
#pragma unroll
  for (int j = 0; j < VEC; ++j) v[j] = prob_of(zt[j], K.c, K.Mt, K.invSt);
  if (nm == 0) return;
  float q[VEC];
#pragma unroll
  for (int j = 0; j < VEC; ++j) q[j] = prob_of(zd[j], K.c, K.Md, K.invSd);
  if (resi) {
    apply_chain_vec<VEC, true>(S2, nm, v, q);
    zero_rejected<VEC>(S2, nm, base, v);
  } else {
    apply_chain_vec<VEC, false>(S2, nm, v, q);
  }
}

// ---------------------------------------------------------------- sampler
// Inverse-CDF draw inside one CTA from fixed-point masses (as the resident
// kernel's sampler): chunk totals locate the chunk that holds the threshold
// `tau` (mass units 2^-44), the chunk's values are written to a free stage
// as fp32, then NW contiguous warp segments, 32 lane ranges and one lane's
// walk find the token.  If rounding leaves tau past the slice's own total,
// the last token with positive mass is taken.  Returns the token's offset in
// the slice (-1 if the slice has no mass).
template <int THREADS, bool BF16>
__device__ int stream_search(Head& H, StreamHead& S2, Ring& R, const VerifyParams& P,
                             const VisitScalars& K, bool resi, size_t off, int lo, int nloc,
                             unsigned long long tau) {
  using G = StreamGeom<THREADS, BF16>;
  constexpr int VEC = G::VEC;
  constexpr int NW = THREADS / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nm = S2.nmaps;
  const int rows = nm > 0 ? 2 : 1;
  if (threadIdx.x == 0) {
    H.misc[0] = -1;  // chunk holding tau
    H.misc[1] = -1;  // last chunk with mass
    H.fixd[0] = 0;   // mass before the chunk
  }
  __syncthreads();
  unsigned long long run = 0;  // thread 0 only
  stream_pass<THREADS, BF16>(R, P, rows, off, nloc,
      [&](const unsigned char* rt, const unsigned char* rd, int k, int clen) -> bool {
        unsigned long long acc = 0;
#pragma unroll
        for (int h = 0; h < G::VPT; ++h) {
          const int g = h * THREADS + (int)threadIdx.x;
          if (g * VEC < clen) {
            float zt[VEC], zd[VEC], v[VEC];
            const int valid = min(VEC, clen - g * VEC);
            load_vec<BF16>(rt, g, valid, zt);
            if (rows == 2) load_vec<BF16>(rd, g, valid, zd);
            else {
#pragma unroll
              for (int j = 0; j < VEC; ++j) zd[j] = -INFINITY;
            }
            final_values<VEC>(S2, K, resi, nm, lo + k * G::CE + g * VEC, zt, zd, v);
#pragma unroll
            for (int j = 0; j < VEC; ++j) acc += to_fix(v[j]);
          }
        }
        acc = warp_sum_u64(acc);
        if (lane == 0) H.seg[warp] = acc;
        __syncthreads();
        if (threadIdx.x == 0) {
          unsigned long long m = 0;
          for (int w = 0; w < NW; ++w) m += H.seg[w];
          if (m > 0) H.misc[1] = k;
          if (H.misc[0] < 0) {
            if (run + m > tau) { H.misc[0] = k; H.fixd[0] = tau - run; }
            else run += m;
          }
        }
        __syncthreads();
        return H.misc[0] >= 0;
      });
  const int kfound = H.misc[0];
  const int klast = H.misc[1];
  if (kfound < 0 && klast < 0) return -1;
  const bool force = kfound < 0;
  const int ks = force ? klast : kfound;
  const unsigned long long t = force ? 0ull : H.fixd[0];
  // Load chunk ks into the next stage, write its values to the stage after.
  const uint32_t slot = R.consumed % (uint32_t)R.S;
  unsigned char* s0 = R.buf + slot * G::SB;
  float* F = reinterpret_cast<float*>(R.buf + ((slot + 1) % (uint32_t)R.S) * G::SB);
  const int clen = min(G::CE, nloc - ks * G::CE);
  constexpr uint32_t es = BF16 ? 2u : 4u;
  {
    const char* st = static_cast<const char*>(P.zt) + (off + (size_t)ks * G::CE) * es;
    const char* sd = static_cast<const char*>(P.zd) + (off + (size_t)ks * G::CE) * es;
    if (R.tma) {
      if (threadIdx.x == 0) {
        const uint32_t bar = R.bar0 + 8u * slot;
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(bar, (uint32_t)rows * (uint32_t)clen * es);
        bulk_g2s(R.addr + slot * G::SB, st, (uint32_t)clen * es, bar);
        if (rows == 2) bulk_g2s(R.addr + slot * G::SB + G::RB, sd, (uint32_t)clen * es, bar);
      }
      R.issued += 1;
      if (R.ok) R.ok = wait_bar(R.bar0 + 8u * slot, (R.consumed / (uint32_t)R.S) & 1u);
      R.consumed += 1;
    } else {
      for (int w = 0; w < rows; ++w) {
        if constexpr (BF16) {
          const uint16_t* src = reinterpret_cast<const uint16_t*>(w ? sd : st);
          uint16_t* dst = reinterpret_cast<uint16_t*>(s0 + w * G::RB);
          for (int i = threadIdx.x; i < clen; i += THREADS) dst[i] = __ldg(src + i);
        } else {
          const float* src = reinterpret_cast<const float*>(w ? sd : st);
          float* dst = reinterpret_cast<float*>(s0 + w * G::RB);
          for (int i = threadIdx.x; i < clen; i += THREADS) dst[i] = __ldg(src + i);
        }
      }
      __syncthreads();
    }
  }
#pragma unroll
  for (int h = 0; h < G::VPT; ++h) {
    const int g = h * THREADS + (int)threadIdx.x;
    float v[VEC];
    if (g * VEC < clen) {
      float zt[VEC], zd[VEC];
      const int valid = min(VEC, clen - g * VEC);
      load_vec<BF16>(s0, g, valid, zt);
      if (rows == 2) load_vec<BF16>(s0 + G::RB, g, valid, zd);
      else {
#pragma unroll
        for (int j = 0; j < VEC; ++j) zd[j] = -INFINITY;
      }
      final_values<VEC>(S2, K, resi, nm, lo + ks * G::CE + g * VEC, zt, zd, v);
    } else {
#pragma unroll
      for (int j = 0; j < VEC; ++j) v[j] = 0.f;
    }
#pragma unroll
    for (int j = 0; j < VEC; ++j) F[g * VEC + j] = v[j];
  }
  __syncthreads();
  // warp segments of SEG elements over the chunk (zeros past clen)
  constexpr int SEG = G::CE / NW;
  {
    const int s0i = warp * SEG;
    unsigned long long acc = 0;
    for (int i = s0i + 4 * lane; i < s0i + SEG; i += 128) {
      const float4 x = *reinterpret_cast<const float4*>(F + i);
      acc += to_fix(x.x) + to_fix(x.y) + to_fix(x.z) + to_fix(x.w);
    }
    acc = warp_sum_u64(acc);
    if (lane == 0) H.seg[warp] = acc;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long a = 0;
    int wstar = -1, last = -1;
    for (int w = 0; w < NW; ++w) {
      const unsigned long long m = H.seg[w];
      if (m > 0) last = w;
      if (!force && wstar < 0) {
        if (a + m > t) wstar = w;
        else a += m;
      }
    }
    const bool f2 = force || wstar < 0;
    H.misc[3] = f2;
    H.misc[2] = f2 ? max(last, 0) : wstar;
    H.fixd[1] = f2 ? 0ull : t - a;
    H.misc[4] = -1;
  }
  __syncthreads();
  if (warp == H.misc[2]) {
    constexpr int SUB = SEG / 32;
    const int r0 = warp * SEG + lane * SUB, r1 = r0 + SUB;
    unsigned long long m = 0;
    int lastpos = -1;
    for (int i = r0; i < r1; ++i) {
      const float x = F[i];
      m += to_fix(x);
      if (x > 0.f) lastpos = i;
    }
    unsigned long long incl = m;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    const unsigned long long tt = H.fixd[1];
    const bool f2 = H.misc[3] != 0;
    const unsigned cross = __ballot_sync(0xffffffffu, !f2 && incl > tt);
    const unsigned pos = __ballot_sync(0xffffffffu, lastpos >= 0);
    const int sel = cross ? __ffs(cross) - 1 : (pos ? 31 - __clz(pos) : 0);
    if (lane == sel) {
      int pick = -1;
      if (cross) {
        const unsigned long long tl = tt - (incl - m);
        unsigned long long a = 0;
        for (int i = r0; i < r1; ++i) {
          a += to_fix(F[i]);
          if (a > tl) { pick = i; break; }
        }
      }
      if (pick < 0) pick = lastpos >= 0 ? lastpos : r0;
      H.misc[4] = pick;
    }
  }
  __syncthreads();
  const int pick = H.misc[4];
  __syncthreads();  // the stage holding F may be refilled afterwards
  return pick < 0 ? -1 : ks * G::CE + pick;
}

// Final draw of a visit: every CTA picks the CTA whose mass range holds
// u * total (as the resident kernel's sampler); that CTA searches its slice.
template <int THREADS, bool BF16>
__device__ bool stream_sample(Head& H, StreamHead& S2, Ring& R, const VerifyParams& P,
                              const VisitScalars& K, bool resi, int mass_kind, const Pending& Pm,
                              float u, int b, int depth, size_t off, int lo, int nloc,
                              uint32_t rank, uint32_t C, int& xp, uint32_t& xph, bool& timeout) {
  using G = StreamGeom<THREADS, BF16>;
  constexpr int VEC = G::VEC;
  constexpr int NW = THREADS / 32;
  const int nm = S2.nmaps;
  const int rows = nm > 0 ? 2 : 1;
  if (P.out_dist || mass_kind == 0) {
    // every CTA: values of its slice (written out when asked) and their sum
    float* dist = P.out_dist ? P.out_dist + (size_t)b * P.V + lo : nullptr;
    float s = 0.f;
    stream_pass<THREADS, BF16>(R, P, rows, off, nloc,
        [&](const unsigned char* rt, const unsigned char* rd, int k, int clen) -> bool {
#pragma unroll
          for (int h = 0; h < G::VPT; ++h) {
            const int g = h * THREADS + (int)threadIdx.x;
            if (g * VEC < clen) {
              float zt[VEC], zd[VEC], v[VEC];
              const int valid = min(VEC, clen - g * VEC);
              load_vec<BF16>(rt, g, valid, zt);
              if (rows == 2) load_vec<BF16>(rd, g, valid, zd);
              else {
#pragma unroll
                for (int j = 0; j < VEC; ++j) zd[j] = -INFINITY;
              }
              final_values<VEC>(S2, K, resi, nm, lo + k * G::CE + g * VEC, zt, zd, v);
#pragma unroll
              for (int j = 0; j < VEC; ++j) {
                s += v[j];
                if (dist && j < valid) dist[k * G::CE + g * VEC + j] = v[j];
              }
            }
          }
          return false;
        });
    if (mass_kind == 0) {
      float o[8];
      int of;
      exchange<NW, false>(H, s, 0.f, 0.f, 0.f, R.ok ? 0 : kFlagTimeout, -1, xp, xph, rank, C, o,
                          of);
      if (of & kFlagTimeout) { timeout = true; return true; }
      mass_kind = 4;
    }
  }
  if (threadIdx.x == 0) {
    unsigned long long total = 0;
    for (uint32_t r = 0; r < C; ++r) total += to_fix(cta_mass(H, r, mass_kind, Pm, K.Mt, K.invSt));
    int cstar = -1;
    unsigned long long before = 0;
    if (total > 0) {
      const unsigned long long kk = (unsigned long long)(u * 16777216.f);
      const unsigned long long lo64 = kk * total, hi64 = __umul64hi(kk, total);
      const unsigned long long tau = (hi64 << 40) | (lo64 >> 24);
      unsigned long long a = 0;
      for (uint32_t r = 0; r < C; ++r) {
        const unsigned long long m = to_fix(cta_mass(H, r, mass_kind, Pm, K.Mt, K.invSt));
        if (a + m > tau) { cstar = (int)r; before = a; break; }
        a += m;
      }
      H.fixd[1] = tau - before;
    }
    H.misc[5] = cstar;
  }
  __syncthreads();
  const int cstar = H.misc[5];
  const unsigned long long tau = H.fixd[1];
  __syncthreads();
  if (cstar < 0) return false;
  if ((int)rank != cstar) return true;
  // A slice whose exchange mass is positive but whose every element rounds
  // to zero mass yields its first token.
  const int pick = stream_search<THREADS, BF16>(H, S2, R, P, K, resi, off, lo, nloc, tau);
  if (threadIdx.x == 0) P.out_tokens[(size_t)b * (P.D + 1) + depth] = lo + max(pick, 0);
  return true;
}

// ---------------------------------------------------------------- kernel
template <int THREADS, bool BF16>
__global__ void __launch_bounds__(THREADS, THREADS >= 512 ? 2 : 4)
    stream_kernel(const VerifyParams P) {
  using G = StreamGeom<THREADS, BF16>;
  constexpr int NW = THREADS / 32;
  constexpr int VEC = G::VEC;
  extern __shared__ __align__(128) unsigned char smem[];
  Head& H = *reinterpret_cast<Head*>(smem);
  StreamHead& S2 = *reinterpret_cast<StreamHead*>(smem + kHeadBytes);
  unsigned char* ring = smem + kHeadBytes + kStreamHeadBytes;
  const int S = P.stages;
  int16_t* par = reinterpret_cast<int16_t*>(ring + (size_t)S * G::SB);
  int16_t* first_child = par + P.npad;
  int16_t* next_sib = first_child + P.npad + 16;
  int32_t* cand_s = reinterpret_cast<int32_t*>(next_sib + P.npad);
  float* u_acc = reinterpret_cast<float*>(cand_s + P.npad);  // [r]: accept test of node r - 1
  float* u_fin = u_acc + P.npad;                             // [r]: final draw at row r

  const int tid = threadIdx.x;
  const uint32_t rank = cluster_ctarank();
  const uint32_t C = cluster_nctarank();
  const int b = (int)cluster_id_x();
  const int N = P.N, V = P.V, D = P.D;
  const int L = P.slice;
  const int lo = (int)rank * L;
  const int nloc = max(0, min(V, lo + L) - lo);
  const bool resi = P.mode == 0;
  const bool bf16 = BF16;

  if (tid < 4) H.pubv[tid] = 0.f;
  if (tid == 0) {
    for (int s = 0; s < S; ++s) mbar_init(smem_addr(&S2.fbar[s]), 1);
    mbar_init(smem_addr(&H.xbar[0]), 1);
    mbar_init(smem_addr(&H.xbar[1]), 1);
    fence_mbar_init();
  }
  for (int i = tid; i < P.npad + 16; i += THREADS) first_child[i] = -1;
  int bad = 0;
  for (int i = tid; i < N; i += THREADS) {
    const int p = __ldg(P.parents + i);
    const bool ok = p >= -1 && p < i;
    bad |= !ok;
    par[i] = (int16_t)(ok ? p : -2);
    cand_s[i] = __ldg(P.cand + (size_t)b * N + i);
  }
  // One Philox block per logit row r: the accept draw of node r - 1 (word 0)
  // and the final draw at row r (word 1).
  for (int r = tid; r <= N; r += THREADS) {
    const U64x4 blk = philox4x64_10((uint64_t)r, (uint64_t)(uint32_t)b, 0, 0, P.seed, 0);
    u_acc[r] = u24(blk.w[0]);
    u_fin[r] = u24(blk.w[1]);
  }
  const bool tree_bad = __syncthreads_or(bad) != 0;
  build_children(par, first_child, next_sib, N);
  __syncthreads();
  cluster_sync();  // every peer has started: its receive slots may now be written

  Ring R;
  R.buf = ring;
  R.addr = smem_addr(ring);
  R.bar0 = smem_addr(&S2.fbar[0]);
  R.S = S;
  R.issued = 0;
  R.consumed = 0;
  R.tma = P.use_tma != 0;
  R.ok = true;

  int err = tree_bad ? kErrTree : 0;
  int info = 0;
  int depth = 0, rejects = 0;
  int node = -1, row = 0;
  uint32_t xph = 0;
  int xp = 0;

  while (!err) {
    const int c1 = first_child[node + 1];
    const bool need_draft = c1 >= 0;
    const size_t rbase = (size_t)b * P.seq_stride + (size_t)row * V;
    const size_t off = rbase + (size_t)lo;

    // children of the node, ascending
    if (tid == 0) {
      int n = 0;
      for (int cn = c1; cn >= 0; cn = next_sib[cn]) {
        if (n == kMaxKids) { n = -1; break; }
        S2.knode[n++] = cn;
      }
      S2.nkids = n;
      S2.nmaps = 0;
    }
    __syncthreads();

    // ---- tempered normaliser (S2): online (reference, sum) per row; the
    // children's tokens' raw logits are read (one thread per child) while
    // the first chunks are in flight
    float mt = -INFINITY, st = 0.f, md = -INFINITY, sd = 0.f;
    stream_pass_pre<THREADS, BF16>(R, P, need_draft ? 2 : 1, off, nloc,
        [&] {
          if (tid < S2.nkids) {
            const int x = cand_s[S2.knode[tid]];
            const bool okx = x >= 0 && x < V;
            S2.kzt[tid] = okx ? raw_logit(P.zt, rbase + (size_t)x, bf16) : 0.f;
            S2.kzd[tid] = okx ? raw_logit(P.zd, rbase + (size_t)x, bf16) : 0.f;
          }
        },
        [&](const unsigned char* rt, const unsigned char* rd, int k, int clen) -> bool {
          float zt[G::VPT * VEC];
#pragma unroll
          for (int h = 0; h < G::VPT; ++h) {
            const int g = h * THREADS + tid;
            float z[VEC];
            if (g * VEC < clen) load_vec<BF16>(rt, g, min(VEC, clen - g * VEC), z);
            else {
#pragma unroll
              for (int j = 0; j < VEC; ++j) z[j] = -INFINITY;
            }
#pragma unroll
            for (int j = 0; j < VEC; ++j) zt[h * VEC + j] = z[j];
          }
          norm_accumulate<G::VPT * VEC>(zt, P.scale_log2, mt, st);
          if (need_draft) {
#pragma unroll
            for (int h = 0; h < G::VPT; ++h) {
              const int g = h * THREADS + tid;
              float z[VEC];
              if (g * VEC < clen) load_vec<BF16>(rd, g, min(VEC, clen - g * VEC), z);
              else {
#pragma unroll
                for (int j = 0; j < VEC; ++j) z[j] = -INFINITY;
              }
#pragma unroll
              for (int j = 0; j < VEC; ++j) zt[h * VEC + j] = z[j];
            }
            norm_accumulate<G::VPT * VEC>(zt, P.scale_log2, md, sd);
          }
          return false;
        });
    const bool bad_t = !(st <= FLT_MAX), bad_d = !(sd <= FLT_MAX);
    const int flags = (bad_t ? kFlagTargetBad : 0) | (bad_d ? kFlagDraftBad : 0) |
                      (R.ok ? 0 : kFlagTimeout);
    float o[8];
    int oflags;
    exchange<NW, true>(H, mt, st, md, sd, flags, -1, xp, xph, rank, C, o, oflags);
    if (oflags & kFlagTimeout) { err |= kErrTimeout; break; }
    if (oflags & kFlagTargetBad) { err |= kErrNonfinite; break; }
    if (o[0] == -INFINITY) { err |= kErrEmpty; break; }
    if (need_draft && (oflags & kFlagDraftBad)) { err |= kErrNonfinite; break; }
    if (need_draft && o[2] == -INFINITY) { err |= kErrEmpty; break; }
    VisitScalars K;
    K.c = P.scale_log2;
    K.Mt = o[0];
    K.invSt = __frcp_rn(o[1]);
    K.Md = o[2];
    K.invSd = need_draft ? __frcp_rn(o[3]) : 0.f;
    Pending Pm{kScale, -1, 0.f, 0.f, 0.f};  // parameters of the latest map (sampler masses)
    int mass_kind = 1;

    if (!need_draft) {
      // accepted leaf (or a root without children): bonus token from p
      bool to = false;
      if (!stream_sample<THREADS, BF16>(H, S2, R, P, K, resi, mass_kind, Pm, u_fin[row], b, depth,
                                        off, lo, nloc, rank, C, xp, xph, to))
        err |= kErrEmpty;
      if (to || !R.ok) err |= kErrTimeout;
      break;
    }
    const int nk = S2.nkids;  // written by thread 0 before the exchange's barriers
    if (nk < 0) { err |= kErrFanout; break; }

    // ---- sequential accept tests over the children (S3), shaping on reject
    int accepted = -1, acc_tok = -1;
    for (int i = 0; i < nk; ++i) {
      const int cn = S2.knode[i];
      const int x = cand_s[cn];
      if (x < 0 || x >= V) { err |= kErrToken; break; }
      const int nm = S2.nmaps;
      const float qx = prob_of(S2.kzd[i], K.c, K.Md, K.invSd);
      float Rx = prob_of(S2.kzt[i], K.c, K.Mt, K.invSt);
      if (resi) {
        Rx = apply_chain<true>(S2, nm, Rx, qx);
        for (int j = 0; j < nm; ++j)
          if (S2.rej[j] == x) Rx = 0.f;
      } else {
        Rx = apply_chain<false>(S2, nm, Rx, qx);
      }
      const float u = u_acc[cn + 1];
      if (__fmul_rn(u, qx) < Rx) { accepted = cn; acc_tok = x; break; }
      rejects += 1;
      float Z = 0.f;
      if (resi) {
        Z = __fsub_rn(qx, Rx);
        if (!(Z > 0.f)) {  // degenerate rejection: R is kept unchanged
          info |= kInfoDegenerate;
          continue;
        }
      }
      if (nm >= kMaxMaps) { err |= kErrFanout; break; }
      // one pass: the residual so far and the sums of the new map
      float s1 = 0.f, s2 = 0.f;
      stream_pass<THREADS, BF16>(R, P, 2, off, nloc,
          [&](const unsigned char* rt, const unsigned char* rd, int k, int clen) -> bool {
#pragma unroll
            for (int h = 0; h < G::VPT; ++h) {
              const int g = h * THREADS + tid;
              if (g * VEC < clen) {
                float zt[VEC], zd[VEC], Rv[VEC], q[VEC];
                const int valid = min(VEC, clen - g * VEC);
                load_vec<BF16>(rt, g, valid, zt);
                load_vec<BF16>(rd, g, valid, zd);
                const int base = lo + k * G::CE + g * VEC;
#pragma unroll
                for (int j = 0; j < VEC; ++j) {
                  Rv[j] = prob_of(zt[j], K.c, K.Mt, K.invSt);
                  q[j] = prob_of(zd[j], K.c, K.Md, K.invSd);
                }
                if (resi) {
                  apply_chain_vec<VEC, true>(S2, nm, Rv, q);
                  zero_rejected<VEC>(S2, nm, base, Rv);
                  const unsigned dx = (unsigned)(x - base);
#pragma unroll
                  for (int j = 0; j < VEC; ++j) {
                    if ((unsigned)j == dx) continue;  // the rejected token: r(x0) = 0
                    const float m = fminf(__fmul_rn(Z, q[j]), Rv[j]);
                    s1 += m;
                    s2 += __fsub_rn(Rv[j], m);
                  }
                } else {
                  apply_chain_vec<VEC, false>(S2, nm, Rv, q);
#pragma unroll
                  for (int j = 0; j < VEC; ++j) s1 += fmaxf(__fsub_rn(Rv[j], q[j]), 0.f);
                }
              }
            }
            return false;
          });
      exchange<NW, false>(H, s1, s2, 0.f, 0.f, R.ok ? 0 : kFlagTimeout, -1, xp, xph, rank, C, o,
                          oflags);
      if (oflags & kFlagTimeout) { err |= kErrTimeout; break; }
      bool has_map = false;
      float a = 0.f, lam = 0.f;
      if (resi) {
        const float S1 = o[0], S2s = o[1];
        const float delta = __fsub_rn(Z, S1);
        lam = S2s > 0.f ? fminf(fmaxf(__fdiv_rn(delta, S2s), 0.f), 1.f) : 0.f;
        const float norm = __fmaf_rn(lam, S2s, S1);
        if (norm > 0.f) {
          has_map = true;
          a = __frcp_rn(norm);
          Pm = Pending{kResi, x, a, Z, lam};
          mass_kind = 2;
        }
      } else if (o[0] > 0.f) {
        has_map = true;
        a = __frcp_rn(o[0]);
        Pm = Pending{kSpec, -1, a, 0.f, 0.f};
        mass_kind = 3;
      }
      if (has_map) {
        if (tid == 0) {
          S2.mZ[nm] = Z;
          S2.mlam[nm] = lam;
          S2.ma[nm] = a;
          S2.rej[nm] = x;
          S2.nmaps = nm + 1;
        }
        __syncthreads();
      } else {
        info |= kInfoDegenerate;
        mass_kind = 0;  // the exchange's partials do not describe R: sum it directly
      }
    }
    if (err) break;

    if (accepted < 0) {
      // every child rejected: residual draw (Algorithm 1, last step)
      bool to = false;
      if (!stream_sample<THREADS, BF16>(H, S2, R, P, K, resi, mass_kind, Pm, u_fin[row], b, depth,
                                        off, lo, nloc, rank, C, xp, xph, to))
        err |= kErrEmpty;
      if (to || !R.ok) err |= kErrTimeout;
      break;
    }
    if (depth >= D) { err |= kErrDepth; break; }
    if (rank == 0 && tid == 0) {
      P.out_tokens[(size_t)b * (D + 1) + depth] = acc_tok;
      if (P.out_nodes) P.out_nodes[(size_t)b * D + depth] = accepted;
    }
    node = accepted;
    row = accepted + 1;
    depth += 1;
    __syncthreads();  // thread 0 rewrites the children list of the next visit
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
  cluster_sync();  // no CTA leaves while a peer may still write its slots
}

}  // namespace rs
