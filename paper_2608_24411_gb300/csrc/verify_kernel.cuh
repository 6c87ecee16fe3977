// Fused verification kernel: one thread-block cluster walks one sequence's
// draft tree (Sec. 3, Algorithm 1, GetProxy).
//
// Data layout on chip.  The vocabulary is cut into C contiguous slices of L
// elements, one per CTA of the cluster.  A slice is a sequence of vectors of
// VEC elements (4 fp32 or 8 bf16 logits = 16 bytes of input); vector g
// belongs to thread g % THREADS in every pass, so per-thread constants stay
// valid across passes.  Each CTA keeps two fp32 rows of its slice in shared
// memory:
//   W  target row: exp((z - m_t) / T), then the current residual R,
//      materialised by every rejection pass,
//   Q  draft row:  exp((z - m_t) / T),
// where m_t is a per-thread exponent reference (the first logit maximum the
// thread saw, raised only when a later logit exceeds it by 64 binary
// orders).  The rows arrive by bulk copy in chunks of 2 * THREADS vectors,
// each with its own mbarrier, and are normalised chunk by chunk while later
// chunks are still in flight; bf16 rows land in the upper half of W / Q and
// are widened in place.  The rows of a node are read from HBM exactly once.
//
// Cluster exchanges.  A visit needs one exchange for the normaliser (online
// max/sum pairs) and one per rejection (two sums).  Each exchange is a push:
// every CTA stores its partial into every peer's receive slot with st.async
// and counts bytes on the peer's mbarrier, so no cluster-wide barrier is
// needed on the hot path.  The owner CTA of the next candidate publishes
// that candidate's stored values in the same exchange, so every CTA
// evaluates the next accept test from bit-identical operands.
//
// Lazy residual.  After rejection j the kernel holds only scalars
// (x0, Z, lambda, 1/norm) of the map R_j -> R_{j+1}; the next pass applies
// it element-wise while it computes the sums of rejection j+1.
#pragma once
#include <cuda_bf16.h>
#include <float.h>
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

// Internal flag bits carried through exchanges.
constexpr int kFlagTargetBad = 1;
constexpr int kFlagDraftBad = 2;
constexpr int kFlagTimeout = 4;

constexpr uint32_t kSpinLimit = 1u << 18;  // suspended try_wait attempts (10 us each) before giving up
constexpr int kMaxCluster = 16;
constexpr int kMaxChunks = 32;             // bulk-copy chunks per row
constexpr int kSlotFloats = 12;
constexpr uint32_t kSlotBytes = 48;
constexpr float kRebaseLog2 = 64.f;        // exponent headroom before a reference moves

struct VerifyParams {
  const void* zt;
  const void* zd;
  const int32_t* parents;  // [N], or [B, N] with parents_stride = N
  const int32_t* cand;
  int32_t* out_tokens;
  int32_t* out_len;
  int32_t* out_nodes;
  float* out_dist;
  int32_t* out_rejects;
  int64_t* out_phase;    // optional [B, 6] cycles per phase (streaming kernel)
  int32_t* draft_out;    // drafting: [B, N] children drawn from q (streaming kernel)
  int32_t* status;
  int64_t seq_stride;  // elements
  int64_t parents_stride;  // elements between sequences' trees (0: one tree)
  uint64_t seed;
  float scale_log2;    // log2(e) / T
  float scale_log2_lo; // log2(e) / T - scale_log2, rounded (SpecInfer instance)
  float exp2_tab[64][2];  // 2^(j / 64), j = -32 .. 31, as double-floats (SpecInfer instance)
  int32_t B, N, V, D;
  int32_t slice;       // L, elements per CTA (multiple of 8)
  int32_t npad;        // padded node count of the tree arrays
  int32_t mode;        // 0 ResiSpec, 1 SpecInfer
  int32_t use_tma;
  int32_t prefetch;    // L2 prefetch of the first child's rows
  int32_t z_applied;   // ResiSpec budget max(Z*, gap) clamped to 1 - R(x0) (streaming kernel)
  int32_t denom_update;  // ResiSpec: each rejection's proxy becomes the test denominator (streaming)
  int32_t level_fill;  // ResiSpec: GetProxy's deficit raises the draft to a level (streaming)
};

struct __align__(16) Slot {
  float v[kSlotFloats];  // [0..3] partials, [4..7] published values, [8] flags, [9] min
};

struct __align__(16) Head {
  unsigned long long tbar[2][kMaxChunks];
  unsigned long long xbar[2];
  Slot rx[2][kMaxCluster];  // receive slots: [exchange parity][source rank]
  float wpart[32][4];       // per-warp partials
  int wflag[32];
  float pubv[4];            // values published by the owner thread of a token
  float bc[kSlotFloats];
  float part[kMaxCluster][4];  // per-CTA partials of the latest exchange
  unsigned long long seg[32];   // sampler: fixed-point warp-segment masses
  unsigned long long fixd[2];   // sampler: fixed-point thresholds
  int misc[8];
};
constexpr int kHeadBytes = 4608;
static_assert(sizeof(Head) <= kHeadBytes, "head too large");

// ---------------------------------------------------------------- residual map
// kScale: R = w * sc with the per-thread scale sc (sc = 1 once R is materialised
// and no map is pending); kResi: GetProxy residual; kSpec: the streaming
// kernel's SpecInfer residual (its sampler masses only).
enum : int { kScale = 0, kResi = 1, kSpec = 2 };

struct Pending {
  int kind;
  int x0;     // rejected token (kResi)
  float a;    // 1 / norm (kResi, kSpec)
  float Z;    // budget (kResi)
  float lam;  // filled fraction of the capacity (kResi)
};

// R_{j+1}(x) from the stored value w = R_j(x) and q(x) = qq; `sc` is the
// per-thread normaliser scale used while the map is still p = w * sc.
// Explicitly rounded intrinsics keep every caller's bits identical.
template <int KIND>
__device__ __forceinline__ float apply_map(const Pending& P, float w, float qq, int idx,
                                           float sc) {
  if constexpr (KIND == kScale) {
    return __fmul_rn(w, sc);
  } else {
    // GetProxy: r = min(Z q, R) + lambda (R - min(Z q, R)) off x0, r(x0) = 0;
    // R' = r / sum r.
    if (idx == P.x0) return 0.f;
    const float m = fminf(__fmul_rn(P.Z, qq), w);
    return __fmul_rn(__fmaf_rn(P.lam, __fsub_rn(w, m), m), P.a);
  }
}

__device__ __forceinline__ float apply_any(const Pending& P, float w, float qq, int idx,
                                           float sc) {
  return P.kind == kScale ? apply_map<kScale>(P, w, qq, idx, sc)
                          : apply_map<kResi>(P, w, qq, idx, sc);
}

// 2^(m - M) / S for a stored reference m in log2 units (0 when m = -inf).
__device__ __forceinline__ float ref_scale(float m, float M, float inv) {
  return m == -INFINITY ? 0.f : __fmul_rn(ex2(__fsub_rn(m, M)), inv);
}

// ---------------------------------------------------------------- reductions
// Butterfly sum over groups of 2^LEVELS lanes (every lane of a group gets the
// same bits).  LEVELS = 5: the whole warp; LEVELS = 4: lanes 0..15 (enough
// for one value per warp of a CTA, or per CTA of a cluster).
template <int LEVELS>
__device__ __forceinline__ float group_sum(float v) {
#pragma unroll
  for (int o = 1 << (LEVELS - 1); o; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// (reference, sum of 2^(z c - reference)) pairs, references in log2 units:
// the common reference is the warp maximum (one redux), each lane rescales
// its sum to it, then a butterfly sum over groups of 2^LEVELS lanes.  Lanes
// that must not contribute hold (-inf, 0).
template <int LEVELS>
__device__ __forceinline__ void pair_reduce(float& m, float& s) {
  const float M = redux_max(m);
  const float t = (m == -INFINITY) ? 0.f : __fmul_rn(s, ex2(__fsub_rn(m, M)));
  s = group_sum<LEVELS>(t);
  m = M;
}

__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity) {
  for (uint32_t it = 0; it < kSpinLimit; ++it)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

// Two-level reduction of per-thread partials, then an all-to-all push of the
// CTA partial to every CTA of the cluster and the same reduction over the C
// received partials.  Every CTA combines identical partials in identical
// lanes, so all CTAs obtain the same bits.
//   NORM: (a0, a1) and (a2, a3) are (reference, scaled sum) pairs of the
//         target and draft rows; SUM: a0, a1 are sums, and a2, a3 too when
//         NSUM = 4 (otherwise they are unused).
//   H.pubv holds the values published by the owner thread of a token; every
//   CTA reads them from the slot of the owner CTA `owner` (-1: none).
//   flags are OR-ed; `mn` is min-reduced over the cluster's CTAs (each CTA
//   passes its own value; the result is left in H.bc[9]).
// out[0..3]: reduced partials, out[4..7]: published values.
template <int NWARPS, bool NORM, int NSUM = 2>
__device__ __forceinline__ void exchange(Head& H, float a0, float a1, float a2, float a3,
                                         int flags, int owner, int& xp, uint32_t& xph,
                                         uint32_t rank, uint32_t C, float (&out)[8],
                                         int& oflags, float mn = INFINITY) {
  static_assert(NWARPS <= 16, "second reduction level covers 16 warps");
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if constexpr (NORM) {
    pair_reduce<5>(a0, a1);
    pair_reduce<5>(a2, a3);
  } else {
    a0 = group_sum<5>(a0);
    a1 = group_sum<5>(a1);
    if constexpr (NSUM > 2) a2 = group_sum<5>(a2);
    if constexpr (NSUM > 3) a3 = group_sum<5>(a3);
  }
  flags = __reduce_or_sync(0xffffffffu, flags);
  if (lane == 0) {
    H.wpart[warp][0] = a0;
    H.wpart[warp][1] = a1;
    H.wpart[warp][2] = a2;
    H.wpart[warp][3] = a3;
    H.wflag[warp] = flags;
  }
  __syncthreads();
  if (warp == 0) {
    const float id = NORM ? -INFINITY : 0.f;
    const bool in = lane < NWARPS;
    a0 = in ? H.wpart[lane][0] : id;
    a1 = in ? H.wpart[lane][1] : 0.f;
    a2 = in ? H.wpart[lane][2] : id;
    a3 = in ? H.wpart[lane][3] : 0.f;
    int f = __reduce_or_sync(0xffffffffu, in ? H.wflag[lane] : 0);
    if constexpr (NORM) {
      pair_reduce<4>(a0, a1);
      pair_reduce<4>(a2, a3);
    } else {
      a0 = group_sum<4>(a0);
      a1 = group_sum<4>(a1);
      if constexpr (NSUM > 2) a2 = group_sum<4>(a2);
      if constexpr (NSUM > 3) a3 = group_sum<4>(a3);
    }
    const int p = xp;
    if (lane < (int)C) {
      const uint32_t dst = map_to_rank(smem_addr(&H.rx[p][rank]), lane);
      const uint32_t bar = map_to_rank(smem_addr(&H.xbar[p]), lane);
      st_async_v4(dst, __float_as_uint(a0), __float_as_uint(a1), __float_as_uint(a2),
                  __float_as_uint(a3), bar);
      st_async_v4(dst + 16, __float_as_uint(H.pubv[0]), __float_as_uint(H.pubv[1]),
                  __float_as_uint(H.pubv[2]), __float_as_uint(H.pubv[3]), bar);
      st_async_v4(dst + 32, (uint32_t)f, __float_as_uint(mn), 0u, 0u, bar);
    }
    if (lane == 0) mbar_arrive_expect_tx(smem_addr(&H.xbar[p]), C * kSlotBytes);
    const bool ok = __all_sync(0xffffffffu, wait_bar(smem_addr(&H.xbar[p]), (xph >> p) & 1u));
    xph ^= 1u << p;
    const bool got = lane < (int)C;
    a0 = got ? H.rx[p][lane].v[0] : id;
    a1 = got ? H.rx[p][lane].v[1] : 0.f;
    a2 = got ? H.rx[p][lane].v[2] : id;
    a3 = got ? H.rx[p][lane].v[3] : 0.f;
    f = __reduce_or_sync(0xffffffffu, got ? __float_as_int(H.rx[p][lane].v[8]) : 0);
    float mr = got ? H.rx[p][lane].v[9] : INFINITY;
#pragma unroll
    for (int o = 8; o; o >>= 1) mr = fminf(mr, __shfl_xor_sync(0xffffffffu, mr, o));
    if (got) {
      H.part[lane][0] = a0; H.part[lane][1] = a1; H.part[lane][2] = a2; H.part[lane][3] = a3;
    }
    if constexpr (NORM) {
      pair_reduce<4>(a0, a1);
      pair_reduce<4>(a2, a3);
    } else {
      a0 = group_sum<4>(a0);
      a1 = group_sum<4>(a1);
      if constexpr (NSUM > 2) a2 = group_sum<4>(a2);
      if constexpr (NSUM > 3) a3 = group_sum<4>(a3);
    }
    if (lane == 0) {
      H.bc[0] = a0; H.bc[1] = a1; H.bc[2] = a2; H.bc[3] = a3;
      const bool has = owner >= 0 && owner < (int)C;
#pragma unroll
      for (int k = 0; k < 4; ++k) H.bc[4 + k] = has ? H.rx[p][owner].v[4 + k] : 0.f;
      H.bc[8] = __int_as_float(f | (ok ? 0 : kFlagTimeout));
      H.bc[9] = mr;
    }
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < 8; ++k) out[k] = H.bc[k];
  oflags = __float_as_int(H.bc[8]);
  xp ^= 1;
}

// ---------------------------------------------------------------- tree
// first_child[n + 1] / next_sibling[c] in ascending node order, built by one
// warp from the highest index down (siblings found with __match_any_sync).
static __device__ void build_children(const int16_t* par, int16_t* first_child, int16_t* next_sib,
                               int N) {
  const int lane = threadIdx.x & 31;
  if ((threadIdx.x >> 5) != 0 || N == 0) return;
  for (int base = (N - 1) & ~31; base >= 0; base -= 32) {
    const int c = base + lane;
    const bool valid = c < N && par[c] >= -1;
    const int key = valid ? par[c] : -1000 - lane;
    const unsigned m = __match_any_sync(0xffffffffu, key);
    const unsigned above = m & ~((2u << lane) - 1u);
    int nxt = -1;
    if (valid) nxt = above ? base + __ffs(above) - 1 : first_child[key + 1];
    __syncwarp();
    if (valid) {
      next_sib[c] = (int16_t)nxt;
      if (lane == __ffs(m) - 1) first_child[key + 1] = (int16_t)c;
    }
    __syncwarp();
  }
}

// ---------------------------------------------------------------- row I/O
// Rows are copied and normalised in chunks of chunk_vectors() 16-byte
// vectors: two per thread for fp32 rows, one per thread for bf16 rows (whose
// widened fp32 values need twice the registers).
template <int THREADS, bool BF16>
__host__ __device__ constexpr int chunk_vectors() { return (BF16 ? 1 : 2) * THREADS; }

// Starts the copies of this CTA's slice [lo, lo + nloc) of the target row
// (and of the draft row when need_draft) that begins at element row_base.
template <int THREADS, bool BF16>
__device__ __forceinline__ void issue_rows(Head& H, const VerifyParams& P, float* W, float* Q,
                                           size_t row_base, bool need_draft, int lo, int nloc) {
  const int L = P.slice;
  const size_t off = row_base + (size_t)lo;
  constexpr uint32_t es = BF16 ? 2u : 4u;
  constexpr uint32_t kChunkBytes = (uint32_t)chunk_vectors<THREADS, BF16>() * 16u;
  // Earlier generic accesses to W / Q must be ordered before the copies.
  fence_proxy_async_smem();
  __syncthreads();
  if (P.use_tma) {
    if (threadIdx.x == 0) {
      const uint32_t bytes = (uint32_t)nloc * es;
      const uint32_t dst_off = BF16 ? 2u * (uint32_t)L : 0u;
      for (int which = 0; which < (need_draft ? 2 : 1); ++which) {
        const char* src = static_cast<const char*>(which ? P.zd : P.zt) + off * es;
        const uint32_t dst = smem_addr(which ? Q : W) + dst_off;
        int k = 0;
        for (uint32_t o = 0; o < bytes; o += kChunkBytes, ++k) {
          const uint32_t n = min(kChunkBytes, bytes - o);
          const uint32_t bar = smem_addr(&H.tbar[which][k]);
          mbar_arrive_expect_tx(bar, n);
          bulk_g2s(dst + o, src + o, n, bar);
        }
      }
    }
  } else {
    for (int which = 0; which < (need_draft ? 2 : 1); ++which) {
      float* dst = which ? Q : W;
      if constexpr (BF16) {
        const uint16_t* src = static_cast<const uint16_t*>(which ? P.zd : P.zt) + off;
        uint16_t* raw = reinterpret_cast<uint16_t*>(dst) + L;
        for (int i = threadIdx.x; i < nloc; i += THREADS) raw[i] = __ldg(src + i);
      } else {
        const float* src = static_cast<const float*>(which ? P.zd : P.zt) + off;
        for (int i = threadIdx.x; i < nloc; i += THREADS) dst[i] = __ldg(src + i);
      }
    }
    __syncthreads();
  }
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Tempered normaliser, first half (S2): one pass over this CTA's slice of
// the target row and (need_draft) the draft row as their chunks land.  With
// c = log2(e) / T and a per-thread reference m per row (log2 units: the
// rounded product of the thread's largest logit so far and c) it stores
// e = 2^(z c - m), one fused multiply-add and one 2^x per element (0 beyond
// the valid part), and returns (m, sum e) per row.  A NaN or +inf logit makes
// the thread's sum non-finite, which is how the error contract detects it.
// Returns false if a chunk wait timed out.
template <int THREADS, bool BF16>
struct RowNorm {
  static constexpr int VEC = BF16 ? 8 : 4;
  static constexpr int CV = chunk_vectors<THREADS, BF16>();  // vectors per chunk
  static constexpr int HV = CV / THREADS;                     // vectors per thread per chunk

  // Load this thread's raw values of chunk k of one row (-inf where invalid).
  __device__ __forceinline__ static void load(const float* buf, int L, int nloc, int k,
                                              float (&z)[HV][VEC]) {
    const int NV = L / VEC, NVV = nloc / VEC;
    const uint16_t* raw = reinterpret_cast<const uint16_t*>(buf) + L;
#pragma unroll
    for (int h = 0; h < HV; ++h) {
      const int g = k * CV + h * THREADS + (int)threadIdx.x;
#pragma unroll
      for (int j = 0; j < VEC; ++j) z[h][j] = -INFINITY;
      if (g < NVV || (g < NV && g * VEC < nloc)) {
        if constexpr (BF16) {
          const uint4 r = *reinterpret_cast<const uint4*>(raw + (size_t)g * 8);
          const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            z[h][2 * j] = bf16_lo(w[j]);
            z[h][2 * j + 1] = bf16_hi(w[j]);
          }
        } else {
          const float4 r = *reinterpret_cast<const float4*>(buf + (size_t)g * 4);
          z[h][0] = r.x; z[h][1] = r.y; z[h][2] = r.z; z[h][3] = r.w;
        }
        if (g >= NVV) {  // ragged tail of the slice (plain-load path only)
#pragma unroll
          for (int j = 0; j < VEC; ++j)
            if (g * VEC + j >= nloc) z[h][j] = -INFINITY;
        }
      }
    }
  }

  // Turn z into e in place, updating (m, s).
  __device__ __forceinline__ static void exps(float* buf, int L, int k, float c,
                                              float (&z)[HV][VEC], float& m, float& s) {
    const int NV = L / VEC;
    float vmax = -INFINITY;
#pragma unroll
    for (int h = 0; h < HV; ++h)
#pragma unroll
      for (int j = 0; j < VEC; ++j) vmax = fmaxf(vmax, z[h][j]);
    if (__fmaf_rn(vmax, c, -m) > kRebaseLog2) {
      // Move this thread's reference up: rescale what it stored so far.
      const float mnew = __fmul_rn(vmax, c);
      if (m != -INFINITY) {
        const float f = ex2(__fsub_rn(m, mnew));
        s = __fmul_rn(s, f);
        for (int k2 = 0; k2 < k; ++k2)
          for (int h = 0; h < HV; ++h) {
            const int g = k2 * CV + h * THREADS + (int)threadIdx.x;
            if (g < NV)
              for (int j = 0; j < VEC; ++j) buf[g * VEC + j] = __fmul_rn(buf[g * VEC + j], f);
          }
      }
      m = mnew;
    }
    if (m == -INFINITY) {  // nothing finite seen yet: every value is -inf or NaN
#pragma unroll
      for (int h = 0; h < HV; ++h)
#pragma unroll
        for (int j = 0; j < VEC; ++j) {
          if (isnan(z[h][j])) s = __int_as_float(0x7fc00000);
          z[h][j] = 0.f;
        }
    } else {
#pragma unroll
      for (int h = 0; h < HV; ++h) {
        float t = 0.f;
#pragma unroll
        for (int j = 0; j < VEC; ++j) {
          z[h][j] = ex2(__fmaf_rn(z[h][j], c, -m));
          t += z[h][j];
        }
        s += t;
      }
    }
  }

  __device__ __forceinline__ static void store(float* buf, int L, int k,
                                               const float (&e)[HV][VEC]) {
    const int NV = L / VEC;
#pragma unroll
    for (int h = 0; h < HV; ++h) {
      const int g = k * CV + h * THREADS + (int)threadIdx.x;
      if (g < NV) {
        float4* d = reinterpret_cast<float4*>(buf + (size_t)g * VEC);
#pragma unroll
        for (int j = 0; j < VEC / 4; ++j)
          d[j] = make_float4(e[h][4 * j], e[h][4 * j + 1], e[h][4 * j + 2], e[h][4 * j + 3]);
      }
    }
  }

  // One row, chunk by chunk as its copies land: returns (mref, sum e) and
  // false if a chunk wait timed out.
  __device__ __forceinline__ static bool row(float* buf, int L, int nloc, float c, uint32_t bar0,
                                             uint32_t parity, int nk_tma, bool wait_tma,
                                             float& m, float& s) {
    const int NK = (L / VEC + CV - 1) / CV;
    bool ok = true;
    m = -INFINITY;
    s = 0.f;
    for (int k = 0; k < NK; ++k) {
      if (wait_tma && k < nk_tma) ok = wait_bar(bar0 + 8u * (uint32_t)k, parity) && ok;
      float z[HV][VEC];
      load(buf, L, nloc, k, z);
      exps(buf, L, k, c, z, m, s);
      if constexpr (BF16) __syncthreads();  // this chunk's raw values are all read
      store(buf, L, k, z);
    }
    return ok;
  }

  // Target row, then (if the node has children) draft row; both rows' copies
  // were issued together, so the draft's chunks land while the target is
  // being normalised.
  __device__ __forceinline__ static bool run(float* W, float* Q, bool need_draft, int L, int nloc,
                                             float c, uint32_t bar_t, uint32_t bar_d,
                                             uint32_t ph_t, uint32_t ph_d, int nk_tma,
                                             bool wait_tma, float& mt, float& st, float& md,
                                             float& sd) {
    bool ok = row(W, L, nloc, c, bar_t, ph_t, nk_tma, wait_tma, mt, st);
    md = -INFINITY;
    sd = 0.f;
    if (need_draft) ok = row(Q, L, nloc, c, bar_d, ph_d, nk_tma, wait_tma, md, sd) && ok;
    return ok;
  }
};

// One rejection pass: materialise R_j = map(W) into W and accumulate the
// sums of rejection j (sum min(Z q, R) and sum (R - min(Z q, R)) over
// x != x0), publishing token xn's values.
// Per-element index tests are needed only in the (at most three) vectors
// that hold x0, xn or the previous map's x0.
template <int VEC, int KIND, bool CHECK>
__device__ __forceinline__ void reject_vector(float (&w)[VEC], const float (&q)[VEC], int base,
                                              const Pending& P, float at, float bt, float mt,
                                              float md, int x0, float Z, int xn, float& t1,
                                              float& t2, float* pubv) {
#pragma unroll
  for (int j = 0; j < VEC; ++j) {
    const int idx = base + j;
    const float qq = __fmul_rn(q[j], bt);
    float R;
    if constexpr (KIND == kResi && !CHECK) {
      const float m = fminf(__fmul_rn(P.Z, qq), w[j]);
      R = __fmul_rn(__fmaf_rn(P.lam, __fsub_rn(w[j], m), m), P.a);
    } else {
      R = apply_map<KIND>(P, w[j], qq, idx, at);
    }
    if (CHECK && idx == xn) { pubv[0] = R; pubv[1] = mt; pubv[2] = q[j]; pubv[3] = md; }
    w[j] = R;
    if (!CHECK || idx != x0) {
      const float m = fminf(__fmul_rn(Z, qq), R);
      t1 += m;
      t2 += __fsub_rn(R, m);
    }
  }
}

template <int THREADS, bool BF16, int KIND>
__device__ __forceinline__ void reject_pass(float* W, const float* Q, int L, int lo,
                                            const Pending& P, float at, float bt, float mt,
                                            float md, int x0, float Z, int xn, float* pubv,
                                            float& s1out, float& s2out) {
  constexpr int VEC = BF16 ? 8 : 4;
  const int NV = L / VEC;
  // vectors that need per-element index tests (-1: none in this slice)
  auto vec_of = [&](int x) { return (x >= lo && x < lo + L) ? (x - lo) / VEC : -1; };
  const int s0 = vec_of(x0), s1 = vec_of(xn), s2 = KIND == kResi ? vec_of(P.x0) : -1;
  float s1sum = 0.f, s2sum = 0.f;
  for (int g = threadIdx.x; g < NV; g += THREADS) {
    float w[VEC], q[VEC];
#pragma unroll
    for (int j = 0; j < VEC / 4; ++j) {
      const float4 a = reinterpret_cast<const float4*>(W + (size_t)g * VEC)[j];
      const float4 b = reinterpret_cast<const float4*>(Q + (size_t)g * VEC)[j];
      w[4 * j] = a.x; w[4 * j + 1] = a.y; w[4 * j + 2] = a.z; w[4 * j + 3] = a.w;
      q[4 * j] = b.x; q[4 * j + 1] = b.y; q[4 * j + 2] = b.z; q[4 * j + 3] = b.w;
    }
    float t1 = 0.f, t2 = 0.f;
    if (g == s0 || g == s1 || g == s2)
      reject_vector<VEC, KIND, true>(w, q, lo + g * VEC, P, at, bt, mt, md, x0, Z, xn, t1, t2,
                                     pubv);
    else
      reject_vector<VEC, KIND, false>(w, q, lo + g * VEC, P, at, bt, mt, md, x0, Z, xn, t1, t2,
                                      pubv);
    s1sum += t1;
    s2sum += t2;
#pragma unroll
    for (int j = 0; j < VEC / 4; ++j)
      reinterpret_cast<float4*>(W + (size_t)g * VEC)[j] =
          make_float4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
  }
  s1out = s1sum;
  s2out = s2sum;
}

// A rejection pass follows either the normaliser scale or a ResiSpec map.
template <int THREADS, bool BF16>
__device__ __forceinline__ void reject_pass_any(float* W, const float* Q, int L, int lo,
                                                const Pending& P, float at, float bt, float mt,
                                                float md, int x0, float Z, int xn, float* pubv,
                                                float& s1, float& s2) {
  if (P.kind == kScale)
    reject_pass<THREADS, BF16, kScale>(W, Q, L, lo, P, at, bt, mt, md, x0, Z, xn, pubv, s1, s2);
  else
    reject_pass<THREADS, BF16, kResi>(W, Q, L, lo, P, at, bt, mt, md, x0, Z, xn, pubv, s1, s2);
}

// ---------------------------------------------------------------- sampler
// The inverse-CDF search runs on exact 64-bit fixed-point masses
// (probability * 2^44, rounded): integer sums are associative, so every
// level of the hierarchical search agrees with every other.

// round(x 2^44) (nearest, ties to even) of a mass x >= 0, with integer
// operations only: the float-to-64-bit-integer conversion runs on the FP64
// pipe, which issues 2 lanes per clock per SM on this part, and the sampler
// converts every element of a slice.  x = m 2^(e - 150) with the 24-bit
// significand m, so x 2^44 = m 2^(e - 106): a left shift when e >= 106,
// else m / 2^s (s = 106 - e) rounded by adding 2^(s-1) - 1 plus the parity
// of the quotient before the shift.  Negative x gives 0 and x >= 2^20
// saturates (neither occurs for masses).
__device__ __forceinline__ unsigned long long to_fix(float x) {
  const uint32_t b = __float_as_uint(x);
  if ((int32_t)b <= 0) return 0ull;
  const int e = (int)(b >> 23);
  const uint32_t m = e ? ((b & 0x7fffffu) | 0x800000u) : b;
  const int sh = (e ? e : 1) - 106;
  if (sh >= 0) return sh >= 40 ? ~0ull : (unsigned long long)m << sh;
  const int s = -sh;
  if (s > 24) return 0ull;
  return (unsigned long long)((m + (1u << (s - 1)) - 1u + ((m >> s) & 1u)) >> s);
}

__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Per-CTA mass of the final distribution, from the partials of the exchange
// that defined it (kind 1: normaliser pairs; 2: ResiSpec sums; 3: SpecInfer
// sums; 4: direct sums).
__device__ __forceinline__ float cta_mass(const Head& H, int r, int kind, const Pending& Pm,
                                          float Mt, float invSt) {
  const float* p = H.part[r];
  switch (kind) {
    case 1: return __fmul_rn(p[1], ref_scale(p[0], Mt, invSt));
    case 2: return __fmul_rn(__fmaf_rn(Pm.lam, p[1], p[0]), Pm.a);
    case 3: return __fmul_rn(p[0], Pm.a);
    default: return p[0];
  }
}

// Inverse-CDF draw: the smallest token x with C(x) > u * C(V-1), u = k 2^-24.
// Every CTA picks the CTA whose mass range holds u * total (masses from the
// exchange partials); that CTA materialises the final distribution in W,
// sums NW contiguous warp segments, then one warp splits its segment into 32
// contiguous lane ranges and one lane walks its range.  When rounding puts
// the threshold past a unit's own total, the search falls back to the last
// token with positive mass, so the result always has R(x) > 0.  Returns
// false when the distribution has no mass.
template <int THREADS, bool BF16>
__device__ bool sample_final(Head& H, const VerifyParams& P, float* W, const float* Q,
                             const Pending& Pm, int mass_kind, float at, float bt, float Mt,
                             float invSt, float u, int b, int depth, int lo, int nloc,
                             uint32_t rank, uint32_t C, int& xp, uint32_t& xph) {
  constexpr int VEC = BF16 ? 8 : 4;
  constexpr int NW = THREADS / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int L = P.slice;
  const int NV = L / VEC;
  bool materialised = false;
  // Owners turn their stored values into the final distribution, in place.
  auto materialise = [&](float* dist) -> float {
    float s = 0.f;
    for (int g = threadIdx.x; g < NV; g += THREADS) {
      float vals[VEC];
#pragma unroll
      for (int j = 0; j < VEC; ++j) {
        const int li = g * VEC + j;
        vals[j] = li < nloc ? apply_any(Pm, W[li], __fmul_rn(Q[li], bt), lo + li, at) : 0.f;
        s += vals[j];
        if (dist && li < nloc) dist[li] = vals[j];
      }
#pragma unroll
      for (int j = 0; j < VEC / 4; ++j)
        reinterpret_cast<float4*>(W + (size_t)g * VEC)[j] =
            make_float4(vals[4 * j], vals[4 * j + 1], vals[4 * j + 2], vals[4 * j + 3]);
    }
    return s;
  };
  const bool need_direct = mass_kind == 0;
  if (P.out_dist || need_direct) {
    const float s = materialise(P.out_dist ? P.out_dist + (size_t)b * P.V + lo : nullptr);
    materialised = true;
    if (need_direct) {
      float o[8];
      int of;
      exchange<NW, false>(H, s, 0.f, 0.f, 0.f, 0, -1, xp, xph, rank, C, o, of);
      mass_kind = 4;
    }
  }
  if (threadIdx.x == 0) {
    unsigned long long total = 0;
    for (uint32_t r = 0; r < C; ++r) total += to_fix(cta_mass(H, r, mass_kind, Pm, Mt, invSt));
    int cstar = -1;
    unsigned long long before = 0;
    if (total > 0) {
      // tau = floor(k * total / 2^24) with u = k / 2^24, exactly
      const unsigned long long k = (unsigned long long)(u * 16777216.f);
      const unsigned long long lo64 = k * total, hi64 = __umul64hi(k, total);
      const unsigned long long tau = (hi64 << 40) | (lo64 >> 24);
      unsigned long long a = 0;
      for (uint32_t r = 0; r < C; ++r) {
        const unsigned long long m = to_fix(cta_mass(H, r, mass_kind, Pm, Mt, invSt));
        if (a + m > tau) { cstar = (int)r; before = a; break; }
        a += m;
      }
      H.fixd[0] = tau - before;
    }
    H.misc[0] = cstar;
  }
  __syncthreads();
  const int cstar = H.misc[0];
  if (cstar < 0) return false;
  if ((int)rank != cstar) return true;

  if (!materialised) {
    materialise(nullptr);
    __syncthreads();
  }
  // warp segments of SEG elements (multiple of 4); W holds 0 beyond nloc
  const int SEG = ((L + NW * 4 - 1) / (NW * 4)) * 4;
  {
    const int s0 = warp * SEG, s1 = min(s0 + SEG, L);
    unsigned long long acc = 0;
    for (int i = s0 + 4 * lane; i < s1; i += 128) {
      const float4 x = *reinterpret_cast<const float4*>(W + i);
      acc += to_fix(x.x) + to_fix(x.y) + to_fix(x.z) + to_fix(x.w);
    }
    acc = warp_sum_u64(acc);
    if (lane == 0) H.seg[warp] = acc;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const unsigned long long t = H.fixd[0];
    unsigned long long a = 0;
    int wstar = -1, last = -1;
    for (int w = 0; w < NW; ++w) {
      const unsigned long long m = H.seg[w];
      if (m > 0) last = w;
      if (a + m > t) { wstar = w; break; }
      a += m;
    }
    H.misc[3] = wstar < 0;  // threshold beyond this CTA's total: take the last token
    H.misc[2] = wstar < 0 ? max(last, 0) : wstar;
    H.fixd[1] = wstar < 0 ? 0 : t - a;
  }
  __syncthreads();
  if (warp == H.misc[2]) {
    const int s0 = warp * SEG, s1 = min(s0 + SEG, L);
    const int SUB = (SEG + 31) / 32;
    const int r0 = s0 + lane * SUB, r1 = min(r0 + SUB, s1);
    unsigned long long m = 0;
    int lastpos = -1;
    for (int i = r0; i < r1; ++i) {
      const float x = W[i];
      m += to_fix(x);
      if (x > 0.f) lastpos = i;
    }
    unsigned long long incl = m;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    const unsigned long long t = H.fixd[1];
    const bool force = H.misc[3] != 0;
    const unsigned cross = __ballot_sync(0xffffffffu, !force && incl > t);
    const unsigned pos = __ballot_sync(0xffffffffu, lastpos >= 0);
    const int sel = cross ? __ffs(cross) - 1 : (pos ? 31 - __clz(pos) : 0);
    if (lane == sel) {
      int pick = -1;
      if (cross) {
        const unsigned long long tl = t - (incl - m);
        unsigned long long a = 0;
        for (int i = r0; i < r1; ++i) {
          a += to_fix(W[i]);
          if (a > tl) { pick = i; break; }
        }
      }
      if (pick < 0) pick = lastpos >= 0 ? lastpos : r0;
      P.out_tokens[(size_t)b * (P.D + 1) + depth] = lo + pick;
    }
  }
  return true;
}

// ---------------------------------------------------------------- kernel
template <int THREADS, bool BF16>
__global__ void __launch_bounds__(THREADS, THREADS >= 512 ? 2 : 3)
    verify_kernel(const VerifyParams P) {
  constexpr int NW = THREADS / 32;
  constexpr int VEC = BF16 ? 8 : 4;
  constexpr uint32_t es = BF16 ? 2u : 4u;
  constexpr uint32_t kChunkBytes = (uint32_t)chunk_vectors<THREADS, BF16>() * 16u;
  extern __shared__ __align__(128) unsigned char smem[];
  Head& H = *reinterpret_cast<Head*>(smem);
  const int L = P.slice;
  float* W = reinterpret_cast<float*>(smem + kHeadBytes);
  float* Q = W + L;
  int16_t* par = reinterpret_cast<int16_t*>(Q + L);
  int16_t* first_child = par + P.npad;
  int16_t* next_sib = first_child + P.npad + 16;
  int32_t* cand_s = reinterpret_cast<int32_t*>(next_sib + P.npad);
  float* u_acc = reinterpret_cast<float*>(cand_s + P.npad);  // [r]: accept test of node r - 1
  float* u_fin = u_acc + P.npad;                             // [r]: final draw at row r

  // Nothing is read before the preceding work on the stream has completed;
  // the next launch may be scheduled from here on (it waits the same way).
  grid_dependency_wait();
  grid_launch_dependents();
  const int tid = threadIdx.x;
  const uint32_t rank = cluster_ctarank();
  const uint32_t C = cluster_nctarank();
  const int b = (int)cluster_id_x();
  const int N = P.N, V = P.V, D = P.D;
  const int lo = (int)rank * L;
  const int nloc = max(0, min(V, lo + L) - lo);
  const int nk_tma = (int)(((uint32_t)nloc * es + kChunkBytes - 1) / kChunkBytes);
  const float c = P.scale_log2;
  // CTA of the cluster whose slice holds token x (-1 for an invalid token)
  auto owner_of = [&](int x) { return (x >= 0 && x < V) ? x / L : -1; };

  if (tid < 4) H.pubv[tid] = 0.f;
  if (tid == 0) {
    for (int w = 0; w < 2; ++w)
      for (int k = 0; k < kMaxChunks; ++k) mbar_init(smem_addr(&H.tbar[w][k]), 1);
    mbar_init(smem_addr(&H.xbar[0]), 1);
    mbar_init(smem_addr(&H.xbar[1]), 1);
    fence_mbar_init();
  }
  __syncthreads();
  // Root rows first: a valid tree with N > 0 always has root children.
  issue_rows<THREADS, BF16>(H, P, W, Q, (size_t)b * P.seq_stride, N > 0, lo, nloc);

  for (int i = tid; i < P.npad + 16; i += THREADS) first_child[i] = -1;
  int bad = 0;
  for (int i = tid; i < N; i += THREADS) {
    const int p = __ldg(P.parents + (size_t)b * P.parents_stride + i);
    const bool ok = p >= -1 && p < i;
    bad |= !ok;
    par[i] = (int16_t)(ok ? p : -2);
    cand_s[i] = __ldg(P.cand + (size_t)b * N + i);
  }
  // Every uniform this sequence can use, off the critical path: one Philox
  // block per logit row r gives the accept draw of node r - 1 (word 0) and
  // the final draw at row r (word 1).
  for (int r = tid; r <= N; r += THREADS) {
    const U64x4 blk = philox4x64_10((uint64_t)r, (uint64_t)(uint32_t)b, 0, 0, P.seed, 0);
    u_acc[r] = u24(blk.w[0]);
    u_fin[r] = u24(blk.w[1]);
  }
  const bool tree_bad = __syncthreads_or(bad) != 0;
  build_children(par, first_child, next_sib, N);
  __syncthreads();
  cluster_sync();  // every peer has started: its receive slots may now be written

  int err = tree_bad ? kErrTree : 0;
  int info = 0;
  int depth = 0, rejects = 0;
  int node = -1, row = 0;
  uint32_t tph = 0, xph = 0;
  int xp = 0;
  uint32_t inflight = N > 0 ? 3u : 1u;  // rows whose copies are not yet consumed

  while (!err) {
    const int c1 = first_child[node + 1];
    const bool need_draft = c1 >= 0;

    // ---- tempered normaliser (S2): one pass per row, then one exchange
    float mref_t, sum_t, mref_d, sum_d;
    const bool ok = RowNorm<THREADS, BF16>::run(
        W, Q, need_draft, L, nloc, c, smem_addr(&H.tbar[0][0]), smem_addr(&H.tbar[1][0]),
        tph & 1u, (tph >> 1) & 1u, nk_tma, P.use_tma, mref_t, sum_t, mref_d, sum_d);
    const bool bad_t = !(sum_t <= FLT_MAX), bad_d = !(sum_d <= FLT_MAX);
    if (ok) {
      tph ^= need_draft ? 3u : 1u;
      inflight = 0;
    }
    const int x1 = need_draft ? cand_s[c1] : -1;
    if (x1 >= lo && x1 < lo + nloc && ((x1 - lo) / VEC) % THREADS == tid) {
      H.pubv[0] = W[x1 - lo];
      H.pubv[1] = mref_t;
      H.pubv[2] = Q[x1 - lo];
      H.pubv[3] = mref_d;
    }
    const int flags = (bad_t ? kFlagTargetBad : 0) | (bad_d ? kFlagDraftBad : 0) |
                      (ok ? 0 : kFlagTimeout);
    float o[8];
    int oflags;
    exchange<NW, true>(H, mref_t, sum_t, mref_d, sum_d, flags, owner_of(x1), xp, xph, rank, C, o,
                       oflags);
    if (oflags & kFlagTimeout) { err |= kErrTimeout; break; }
    if (oflags & kFlagTargetBad) { err |= kErrNonfinite; break; }
    if (o[0] == -INFINITY) { err |= kErrEmpty; break; }
    if (need_draft && (oflags & kFlagDraftBad)) { err |= kErrNonfinite; break; }
    if (need_draft && o[2] == -INFINITY) { err |= kErrEmpty; break; }
    const float Mt = o[0], invSt = __frcp_rn(o[1]);
    const float Md = o[2], invSd = need_draft ? __frcp_rn(o[3]) : 0.f;
    float at = ref_scale(mref_t, Mt, invSt);  // 1 once R is materialised with no map pending
    bool ident = false;
    const float bt = need_draft ? ref_scale(mref_d, Md, invSd) : 0.f;
    float pub[4] = {o[4], o[5], o[6], o[7]};
    Pending Pm{kScale, -1, 0.f, 0.f, 0.f};
    int mass_kind = 1;

    if (!need_draft) {
      // accepted leaf (or a root without children): bonus token from p
      if (!sample_final<THREADS, BF16>(H, P, W, Q, Pm, mass_kind, at, bt, Mt, invSt, u_fin[row],
                                       b, depth, lo, nloc, rank, C, xp, xph))
        err |= kErrEmpty;
      break;
    }
    if (P.prefetch && tid == 0) {
      // The first child is the most likely to be accepted: warm L2 with its rows.
      const size_t base = ((size_t)b * P.seq_stride + (size_t)(c1 + 1) * V + lo) * es;
      const uint32_t bytes = (uint32_t)nloc * es;
      const int nrows = first_child[c1 + 1] >= 0 ? 2 : 1;
      for (int w = 0; w < nrows; ++w) {
        const char* src = static_cast<const char*>(w ? P.zd : P.zt) + base;
        for (uint32_t o2 = 0; o2 < bytes; o2 += kChunkBytes)
          prefetch_l2(src + o2, min(kChunkBytes, bytes - o2));
      }
    }

    // ---- sequential accept tests over the children (S3), shaping on reject
    int accepted = -1, acc_tok = -1;
    for (int cn = c1; cn >= 0;) {
      const int x = cand_s[cn];
      if (x < 0 || x >= V) { err |= kErrToken; break; }
      const float qx = __fmul_rn(pub[2], ref_scale(pub[3], Md, invSd));
      const float Rx = Pm.kind != kScale ? apply_any(Pm, pub[0], qx, x, 0.f)
                       : ident          ? pub[0]
                                        : __fmul_rn(pub[0], ref_scale(pub[1], Mt, invSt));
      const float u = u_acc[cn + 1];
      if (__fmul_rn(u, qx) < Rx) { accepted = cn; acc_tok = x; break; }
      rejects += 1;
      const int nxt = next_sib[cn];
      const int xn = nxt >= 0 ? cand_s[nxt] : -1;
      float s1 = 0.f, s2 = 0.f;
      // ResiSpec rejection (Algorithm 1, GetProxy); SpecInfer runs on the
      // streaming kernel
      const float Z = __fsub_rn(qx, Rx);
      if (!(Z > 0.f)) {
        // degenerate rejection: keep R, fetch the next candidate's values
        info |= kInfoDegenerate;
        if (xn >= lo && xn < lo + nloc && ((xn - lo) / VEC) % THREADS == tid) {
          H.pubv[0] = W[xn - lo];
          H.pubv[1] = mref_t;
          H.pubv[2] = Q[xn - lo];
          H.pubv[3] = mref_d;
        }
        exchange<NW, false>(H, 0.f, 0.f, 0.f, 0.f, 0, owner_of(xn), xp, xph, rank, C, o,
                            oflags);
        if (oflags & kFlagTimeout) { err |= kErrTimeout; break; }
        pub[0] = o[4]; pub[1] = o[5]; pub[2] = o[6]; pub[3] = o[7];
        mass_kind = 0;
        cn = nxt;
        continue;
      }
      reject_pass_any<THREADS, BF16>(W, Q, L, lo, Pm, at, bt, mref_t, mref_d, x, Z, xn, H.pubv,
                                     s1, s2);
      exchange<NW, false>(H, s1, s2, 0.f, 0.f, 0, owner_of(xn), xp, xph, rank, C, o,
                          oflags);
      if (oflags & kFlagTimeout) { err |= kErrTimeout; break; }
      const float S1 = o[0], S2 = o[1];
      const float delta = __fsub_rn(Z, S1);
      const float lam = S2 > 0.f ? fminf(fmaxf(__fdiv_rn(delta, S2), 0.f), 1.f) : 0.f;
      const float norm = __fmaf_rn(lam, S2, S1);
      if (norm > 0.f) {
        Pm = Pending{kResi, x, __frcp_rn(norm), Z, lam};
        mass_kind = 2;
      } else {  // R_j is materialised in W: continue from it unchanged
        Pm = Pending{kScale, -1, 1.f, 0.f, 0.f};
        at = 1.f;
        ident = true;
        info |= kInfoDegenerate;
        mass_kind = 0;
      }
      pub[0] = o[4]; pub[1] = o[5]; pub[2] = o[6]; pub[3] = o[7];
      cn = nxt;
    }
    if (err) break;

    if (accepted < 0) {
      // every child rejected: residual draw (Algorithm 1, last step)
      if (!sample_final<THREADS, BF16>(H, P, W, Q, Pm, mass_kind, at, bt, Mt, invSt, u_fin[row],
                                       b, depth, lo, nloc, rank, C, xp, xph))
        err |= kErrEmpty;
      break;
    }
    if (depth >= D) { err |= kErrDepth; break; }
    node = accepted;
    row = accepted + 1;
    issue_rows<THREADS, BF16>(H, P, W, Q, (size_t)b * P.seq_stride + (size_t)row * V,
                              first_child[node + 1] >= 0, lo, nloc);
    inflight = first_child[node + 1] >= 0 ? 3u : 1u;
    if (rank == 0 && tid == 0) {
      P.out_tokens[(size_t)b * (D + 1) + depth] = acc_tok;
      if (P.out_nodes) P.out_nodes[(size_t)b * D + depth] = accepted;
    }
    depth += 1;
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
  if (inflight && P.use_tma && tid == 0) {
    // copies issued but never consumed (bad tree, timeout): let them land
    // (bounded) before the CTA's shared memory is released
    for (int k = 0; k < nk_tma; ++k) {
      if (inflight & 1u) wait_bar(smem_addr(&H.tbar[0][k]), tph & 1u);
      if (inflight & 2u) wait_bar(smem_addr(&H.tbar[1][k]), (tph >> 1) & 1u);
    }
  }
  cluster_sync();  // no CTA leaves while a peer may still write its slots
}

}  // namespace rs
