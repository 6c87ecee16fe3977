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
// streams it in chunks of 8 logits per thread and row (two 16-byte fp32
// vectors or one bf16 vector).  Every thread copies its own vectors of the
// next S - 1 chunks into its own slots of a shared-memory ring with
// cp.async (16-byte asynchronous copies) and reads back only what it copied
// itself, so no barrier is needed between chunks and the bytes in flight
// cost no registers.  With two 512-thread or three 256-thread CTAs per SM
// this saturates HBM, and one
// CTA alone streams about twice as fast as through a bulk-copy (TMA) ring
// of the same size, whose single issuing thread and per-chunk barrier
// limit it.  A visit runs
//   NORM   online (reference, sum) of 2^(z c) per thread, c = log2(e) / T,
//          then one cluster exchange gives the global (M, S) of each row;
//   REJ    once per rejected candidate (Algorithm 1, GetProxy / Eq. 2):
//          recomputes p = 2^(z_t c - M_t) / S_t and q likewise from the raw
//          logits (L2 hits), applies the residual maps of the earlier
//          rejections in order, and sums the terms of the new map;
//   SAMP   residual or bonus draw, in the CTA that holds the threshold.
// After the normaliser every value is a function of the raw logit and
// cluster-wide scalars only, so any thread may compute any element and every
// CTA evaluates the accept tests itself from the candidates' raw logits.
#pragma once
#include <type_traits>

#include "specinfer.cuh"
#include "verify_kernel.cuh"

namespace rs {

constexpr int kMaxMaps = 128;          // residual maps per node (rejections with a map)
// Phases of the optional per-sequence cycle counters: setup, normaliser
// passes, normaliser exchanges, accept tests and budgets (the paper's
// "budgeting"), rejection passes with their exchanges ("redistribution"; the
// proxy is never materialised), the final draw.
enum : int { kPhaseSetup = 0, kPhaseNorm, kPhaseNormX, kPhaseTest, kPhaseRej, kPhaseDraw, kPhases };
constexpr int kMaxKids = kMaxMaps;      // children per node the streaming kernel walks
static_assert(2 * kMaxKids <= 256, "per-visit loads and draws use distinct threads of a CTA");
constexpr int kErrFanout = 64;

// ResiSpec residual maps are kept in unnormalised units.  With
// p~ = 2^(z_t c - M_t) and q~ = 2^(z_d c - M_d) (so p = p~ / S_t,
// q = q~ / S_d), the residual after i maps is R_i = sigma_i R~_i, R~_0 = p~,
// sigma_0 = 1 / S_t, and map i (Z_i, lambda_i, normaliser 1 / a_i) becomes,
// element-wise, m = min(k_i q~, R~), R~' = m + lambda_i (R~ - m), with
// k_i = Z_i / (S_d sigma_{i-1}) and sigma_i = sigma_{i-1} a_i: every scale is
// folded into the per-map scalar k_i and the running factor sigma.  (The
// SpecInfer recurrence needs no list of maps: specinfer.cuh.)  The form keeps
// m (its minimum taken directly) and R~ - m separate: folding the map into
// R~ - (1 - lambda_i)(R~ - m) would round 1 - lambda_i, an error that the
// renormalisation by a small Z_i magnifies wherever m + lambda_i (R~ - m)
// is much smaller than R~.  Maps are applied two lanes per instruction.
struct __align__(16) StreamHead {
  float2 map[kMaxMaps];  // {k_i, lambda_i} of map i
  union {
    float mdsc[kMaxMaps];     // scale of the test denominator's D~ after map i
    float tab[kExp2Tab][2];   // SpecInfer instance: 2^(j/64) as double-floats
  };
  int rej[kMaxMaps];     // rejected tokens (ResiSpec: their residual is 0)
  int16_t rejk[kMaxMaps];  // their child index in this visit
  float kzt[kMaxKids];   // raw target / draft logits of the children's tokens
  float kzd[kMaxKids];
  float kua[kMaxKids];   // their accept draws U(seed, b, child + 1, 0)
  float ufin;            // the visit's final draw U(seed, b, row, 1)
  int nmaps;
  // Chunk records of the pass that defines the visit's final distribution
  // (see ChunkRec): two floats per (chunk, warp), chunk-major.
  float crec[2][256];
  // optional phase counters (clock64 cycles, thread 0): see kPhase*
  unsigned long long phc[kPhases];
  unsigned long long ph_last;
  int ph_cur;
};
constexpr int kStreamHeadBytes = 6144;
constexpr int kMaxChunkRecs = 256;  // (chunk, warp) records per CTA
static_assert(sizeof(StreamHead) <= kStreamHeadBytes, "stream head too large");

// Eight logits per thread, chunk and row (one 16-byte vector of bf16, two
// of fp32), and as many ring stages as fit 96 KB at 512 threads (6 for bf16,
// 3 for fp32).  One fp32 vector per thread and 6 stages of 16 KB, more
// copies in flight, measured 9 % slower on the fp32 workload: the pass
// loop's fixed cost per chunk then falls on four elements instead of eight.
template <int THREADS, bool BF16>
struct StreamGeom {
  static constexpr int VEC = BF16 ? 8 : 4;            // elements per 16-byte vector
  static constexpr int VPT = BF16 ? 1 : 2;            // vectors per thread per chunk and row
  static constexpr int NE = VPT * VEC;                // elements per thread per chunk and row
  static constexpr int NP = NE / 2;                   // their pairs (packed arithmetic)
  static constexpr int CE = NE * THREADS;             // elements per chunk and row
  static constexpr uint32_t RB = (uint32_t)VPT * THREADS * 16u;  // bytes per chunk and row
  static constexpr uint32_t SB = 2u * RB;             // bytes per ring stage (target, draft)
  static constexpr int S = (96 * 1024 * THREADS / 512) / SB;  // ring stages
  static constexpr uint32_t RING = S * SB;
};

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// The rows one pass streams: element 0 of the CTA's slice in each row.
struct Src {
  const char* t;  // target row
  const char* d;  // draft row (rows == 2)
  int rows;
  int nloc;
  bool vec;       // 16-byte aligned rows: vector loads
  bool held;      // every chunk of these rows is in ring stage k (slice <= S chunks)
};

template <bool BF16>
__device__ __forceinline__ uint4 neg_inf_vec() {
  const uint32_t w = BF16 ? 0xff80ff80u : 0xff800000u;
  return make_uint4(w, w, w, w);
}

// The VEC values of one 16-byte vector.
template <bool BF16>
__device__ __forceinline__ void unpack_vec(const uint4& w, float (&z)[BF16 ? 8 : 4]) {
  const uint32_t v[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if constexpr (BF16) {
      z[2 * i] = bf16_lo(v[i]);
      z[2 * i + 1] = bf16_hi(v[i]);
    } else {
      z[i] = __uint_as_float(v[i]);
    }
  }
}

// Vector h of this thread in a ring stage row: slice element
// k CE + (h THREADS + tid) VEC of chunk k.  Vectors past the slice hold
// -inf (written by the copy step).
__device__ __forceinline__ uint4 stage_vec(const unsigned char* row, int h, int threads) {
  return reinterpret_cast<const uint4*>(row)[h * threads + (int)threadIdx.x];
}

// Element j (0 <= j < NE) of this thread's chunk in a ring stage row.
template <int THREADS, bool BF16>
__device__ __forceinline__ float stage_elem(const unsigned char* row, int j) {
  constexpr int VEC = BF16 ? 8 : 4;
  const unsigned char* v =
      row + ((j / VEC) * THREADS + (int)threadIdx.x) * 16 + (j % VEC) * (BF16 ? 2 : 4);
  if constexpr (BF16)
    return __uint_as_float((uint32_t)*reinterpret_cast<const unsigned short*>(v) << 16);
  else
    return *reinterpret_cast<const float*>(v);
}

template <int THREADS, bool BF16>
struct StageElem {
  const unsigned char* row;
  __device__ __forceinline__ float operator()(int j) const {
    return stage_elem<THREADS, BF16>(row, j);
  }
};

// This thread's vectors of a ring stage row, kept packed; element j for a
// compile-time j.
template <int THREADS, bool BF16>
struct ChunkRegs {
  static constexpr int VPT = StreamGeom<THREADS, BF16>::VPT;
  uint4 w[VPT];
  __device__ __forceinline__ explicit ChunkRegs(const unsigned char* row) {
#pragma unroll
    for (int h = 0; h < VPT; ++h) w[h] = stage_vec(row, h, THREADS);
  }
  __device__ __forceinline__ float operator()(int j) const {
    constexpr int VEC = BF16 ? 8 : 4;
    const uint4& v = w[j / VEC];
    const int e = j % VEC;
    if constexpr (BF16) {
      const uint32_t x = (e >> 1) == 0 ? v.x : (e >> 1) == 1 ? v.y : (e >> 1) == 2 ? v.z : v.w;
      return (e & 1) ? bf16_hi(x) : bf16_lo(x);
    } else {
      return __uint_as_float(e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w);
    }
  }
};

// This thread's NE values of a ring stage row as NP = NE / 2 pairs, in the
// order of its vectors (pair j holds elements 2j, 2j + 1 of the thread's chunk).
template <int THREADS, bool BF16>
__device__ __forceinline__ void load_pairs(const unsigned char* row,
                                           float2 (&z)[StreamGeom<THREADS, BF16>::NP]) {
  using G = StreamGeom<THREADS, BF16>;
#pragma unroll
  for (int h = 0; h < G::VPT; ++h) {
    const uint4 w = stage_vec(row, h, THREADS);
    if constexpr (BF16) {
      const uint32_t v[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) z[4 * h + i] = make_float2(bf16_lo(v[i]), bf16_hi(v[i]));
    } else {
      z[2 * h] = make_float2(__uint_as_float(w.x), __uint_as_float(w.y));
      z[2 * h + 1] = make_float2(__uint_as_float(w.z), __uint_as_float(w.w));
    }
  }
}

// Ring layout of a pass: a pass over both rows keeps S stages of SB bytes
// (target row, then draft row); a pass over the target row alone keeps 2 S
// stages of RB bytes, twice as many chunks in flight.  Chunk k of a pass
// lives in stage k mod depth.  The layout is chosen at run time, so each
// pass body is compiled once.
template <int THREADS, bool BF16>
__device__ __forceinline__ int ring_depth(bool two) {
  using G = StreamGeom<THREADS, BF16>;
  return two ? G::S : 2 * G::S;
}
template <int THREADS, bool BF16>
__device__ __forceinline__ uint32_t ring_stride(bool two) {
  using G = StreamGeom<THREADS, BF16>;
  return two ? G::SB : G::RB;
}

// Copies this thread's vectors of chunk k into ring stage `st` (the copies
// of one chunk form one cp.async group): the target row, and the draft row
// RB bytes further when `two`.  Aligned rows: 16-byte asynchronous copies;
// other rows: element loads stored synchronously.
template <int THREADS, bool BF16>
__device__ __forceinline__ void copy_chunk(const Src& s, int k, unsigned char* st, bool two) {
  using G = StreamGeom<THREADS, BF16>;
  constexpr int VEC = G::VEC;
  constexpr int es = BF16 ? 2 : 4;
  const uint4 ninf = neg_inf_vec<BF16>();
#pragma unroll
  for (int h = 0; h < G::VPT; ++h) {
    const int g = h * THREADS + (int)threadIdx.x;
    const int e0 = k * G::CE + g * VEC;
    uint4* dt = reinterpret_cast<uint4*>(st) + g;
    uint4* dd = reinterpret_cast<uint4*>(st + G::RB) + g;
    if (s.vec) {
      // nloc is a multiple of VEC on this path: a vector is whole or absent
      if (e0 < s.nloc) {
        cp_async16(dt, s.t + (size_t)e0 * es);
        if (two) cp_async16(dd, s.d + (size_t)e0 * es);
      } else {
        *dt = ninf;
        if (two) *dd = ninf;
      }
    } else {
      uint32_t wt[4], wd[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if constexpr (BF16) {
          uint32_t lt[2], ld[2];
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            const int e = e0 + 2 * i + j;
            const bool in = e < s.nloc;
            lt[j] = in ? (uint32_t)__ldg(reinterpret_cast<const uint16_t*>(s.t) + e) : 0xff80u;
            ld[j] = (two && in) ? (uint32_t)__ldg(reinterpret_cast<const uint16_t*>(s.d) + e)
                                : 0xff80u;
          }
          wt[i] = lt[0] | (lt[1] << 16);
          wd[i] = ld[0] | (ld[1] << 16);
        } else {
          const int e = e0 + i;
          const bool in = e < s.nloc;
          wt[i] = in ? __float_as_uint(__ldg(reinterpret_cast<const float*>(s.t) + e))
                     : 0xff800000u;
          wd[i] = (two && in) ? __float_as_uint(__ldg(reinterpret_cast<const float*>(s.d) + e))
                              : 0xff800000u;
        }
      }
      *dt = make_uint4(wt[0], wt[1], wt[2], wt[3]);
      if (two) *dd = make_uint4(wd[0], wd[1], wd[2], wd[3]);
    }
  }
  cp_async_commit();
}

// Chunk k's stage when the slice is held in the ring (see Src::held).
template <int THREADS, bool BF16>
__device__ __forceinline__ unsigned char* held_stage(unsigned char* ring, const Src& s, int k) {
  return ring + (size_t)k * ring_stride<THREADS, BF16>(s.rows == 2);
}

// Streams the slice chunk by chunk, depth - 1 chunks ahead (the layout
// above), calling body(target_stage_row, draft_stage_row, k) with all
// threads (the draft pointer is meaningful only for passes over both rows);
// body returns true (uniformly) to end the pass.  pre() runs once, after the
// first copies are issued.  On return every copy of the pass has landed.
// A pass issues its first copies when it starts: issuing them earlier, during
// the cluster exchange before it, measured slower (113 against 108 us on the
// fp32 binary-tree workload), since after an accepted test the copies were
// for rows no pass would read, and the next visit had to wait for them.
// ROWS: 2 or 1 when the caller knows s.rows, 0 to read it.
template <int THREADS, bool BF16, int ROWS = 0, class Pre, class Body>
__device__ __forceinline__ void stream_pass_pre(unsigned char* ring, const Src& s, Pre&& pre,
                                                Body&& body) {
  using G = StreamGeom<THREADS, BF16>;
  const int NK = (s.nloc + G::CE - 1) / G::CE;
  if (s.held) {  // the rows stayed in the ring since the visit's first pass
    pre();
    for (int k = 0; k < NK; ++k) {
      const unsigned char* st = held_stage<THREADS, BF16>(ring, s, k);
      if (body(st, st + G::RB, k)) break;
    }
    return;
  }
  const bool two = ROWS == 2 || (ROWS == 0 && s.rows == 2);
  const int S = ring_depth<THREADS, BF16>(two);
  const uint32_t stride = ring_stride<THREADS, BF16>(two);
  for (int k = 0; k < S - 1; ++k) {
    if (k < NK) copy_chunk<THREADS, BF16>(s, k, ring + k * stride, two);
    else cp_async_commit();
  }
  pre();
  int slot = 0;
  for (int k = 0; k < NK; ++k) {
    const int kn = k + S - 1;
    const int nslot = slot == 0 ? S - 1 : slot - 1;  // (k + S - 1) % S
    if (kn < NK) copy_chunk<THREADS, BF16>(s, kn, ring + nslot * stride, two);
    else cp_async_commit();
    // chunk k's copies (this thread's) have landed
    if (two) cp_async_wait<G::S - 1>();
    else cp_async_wait<2 * G::S - 1>();
    const unsigned char* st = ring + slot * stride;
    const bool stop = body(st, st + G::RB, k);
    slot = slot == S - 1 ? 0 : slot + 1;
    if (stop) break;
  }
  cp_async_wait<0>();
}

template <int THREADS, bool BF16, int ROWS = 0, class Body>
__device__ __forceinline__ void stream_pass(unsigned char* ring, const Src& s, Body&& body) {
  stream_pass_pre<THREADS, BF16, ROWS>(ring, s, [] {}, body);
}

__device__ __forceinline__ float raw_logit(const void* base, size_t i, bool bf16) {
  if (bf16) {
    const uint16_t h = __ldg(static_cast<const uint16_t*>(base) + i);
    return __uint_as_float((uint32_t)h << 16);
  }
  return __ldg(static_cast<const float*>(base) + i);
}

// Online (reference, sum) of 2^(z c) over one thread's values of a chunk,
// for one or two rows at once (independent chains for the scheduler).  The
// reference m (log2 units) starts at the sentinel -FLT_MAX and is raised to
// the rounded product of the largest logit and c whenever a value exceeds
// it; the sum is rescaled.  Tracking the maximum exactly keeps every 2^x
// argument at or below 0, where its rounding is below 2^-24 absolute: a
// reference lagging by d binary orders would cost up to d 2^-24 relative
// error in each term, and the later passes compute p from the exact global
// maximum, so the two would drift apart.  With the sentinel no branch is
// needed for rows that are all -inf so far (2^(-inf) = 0), and NaN or +inf
// still makes the sum non-finite (detected by the caller).
constexpr float kNoRef = -FLT_MAX;

template <int NP>
__device__ __forceinline__ float max_pairs(const float2 (&z)[NP]) {
  if constexpr (NP == 4) {
    return fmax3(fmax3(z[0].x, z[0].y, z[1].x), fmax3(z[1].y, z[2].x, z[2].y),
                 fmaxf(z[3].x, z[3].y));
  } else {
    static_assert(NP == 2, "two or four pairs per chunk");
    return fmax3(fmax3(z[0].x, z[0].y, z[1].x), z[1].y, -INFINITY);
  }
}

// Sum of NP pairs, pairwise.
template <int NP>
__device__ __forceinline__ float2 sum_pairs(const float2 (&a)[NP]) {
  if constexpr (NP == 4) return __fadd2_rn(__fadd2_rn(a[0], a[1]), __fadd2_rn(a[2], a[3]));
  else return __fadd2_rn(a[0], a[1]);
}

// Smallest z_t - z_d of a chunk's pairs (the Z_applied bound min p / q is
// 2^((z_t - z_d) c) scaled by row constants, so it is taken on the logit
// difference).  A token with q = 0 (z_d = -inf) gives +inf and a padding
// slot (both -inf) NaN; both are ignored by the minimum.
template <int NP>
__device__ __forceinline__ float dmin_pairs(const float2 (&zt)[NP], const float2 (&zd)[NP]) {
  float m = INFINITY;
#pragma unroll
  for (int j = 0; j < NP; ++j) {
    const float2 d = __ffma2_rn(zd[j], dup2(-1.f), zt[j]);
    m = fminf(m, fminf(d.x, d.y));
  }
  return m;
}

__device__ __forceinline__ void rebase2(float vmax, float c, float& m, float2& s) {
  const float mnew = __fmul_rn(vmax, c);
  s = __fmul2_rn(s, dup2(ex2(__fsub_rn(m, mnew))));  // 0 from the sentinel
  m = mnew;
}

// Sum of 2^(z c - m) over a chunk's pairs, as a pair of partial sums.
template <int NP>
__device__ __forceinline__ float2 exp_sum(const float2 (&z)[NP], float2 c2, float2 nm2) {
  float2 e[NP];
#pragma unroll
  for (int j = 0; j < NP; ++j) e[j] = ex2x2(__ffma2_rn(z[j], c2, nm2));
  return sum_pairs<NP>(e);
}

// One chunk of a thread's values into its online (reference, sum) pairs;
// the sums are kept as pairs of lanes.  Returns the chunk's own target terms
// (and, TWO, its draft terms in dpart).
template <bool TWO, int NP>
__device__ __forceinline__ float2 norm_accumulate(const float2 (&zt)[NP], const float2 (&zd)[NP],
                                                  float c, float& mt, float2& st, float& md,
                                                  float2& sd, float2& dpart) {
  const float vt = max_pairs<NP>(zt);
  const bool rt = __fmaf_rn(vt, c, -mt) > 0.f;
  float vd = 0.f;
  bool rd = false;
  if constexpr (TWO) {
    vd = max_pairs<NP>(zd);
    rd = __fmaf_rn(vd, c, -md) > 0.f;
  }
  if (rt || rd) {  // rare: a new reference for one of the rows
    if (rt) rebase2(vt, c, mt, st);
    if constexpr (TWO)
      if (rd) rebase2(vd, c, md, sd);
  }
  const float2 c2 = dup2(c);
  const float2 part = exp_sum<NP>(zt, c2, dup2(-mt));  // this chunk's target terms
  st = __fadd2_rn(st, part);
  if constexpr (TWO) {
    dpart = exp_sum<NP>(zd, c2, dup2(-md));  // and its draft terms
    sd = __fadd2_rn(sd, dpart);
  }
  return part;
}

// Chunk records: the pass that defines a visit's final distribution leaves,
// per chunk of the slice and warp, the warp's share of that distribution's
// mass, so that the final draw finds the chunk holding its threshold
// without another pass over the slice.  The mass of chunk k is
//   kind 1 (a leaf's normaliser: the bonus draw samples p; or, when the
//           kernel drafts, the draft row q):
//     sum_w rec1[k, w] 2^(rec0[k, w] - a) b   (warp reference, warp sum;
//                                              a = M, b = 1 / S)
//   kind 2 (the last ResiSpec rejection: R~' = m + lambda t):
//     sum_w (rec0[k, w] + a rec1[k, w]) b     (a = lambda, b = sigma)
//   kind 3 (the last SpecInfer rejection): sum_w rec0[k, w] b   (b = 1 / T)
// in fixed warp order (deterministic).  Records exist when the slice has at
// most kMaxChunkRecs / NW chunks; kind 0: none (the draw runs a pass).
struct ChunkRec {
  int kind;
  float a, b;
};

// Cluster-wide scalars of a visit after the normaliser.
static_assert(sizeof(VerifyParams::exp2_tab) == sizeof(float) * 2 * kExp2Tab &&
                  sizeof(float) * 2 * kExp2Tab <= sizeof(float) * kMaxMaps,
              "exp2 table size");

struct VisitScalars {
  float c;           // log2(e) / T
  float Mt, invSt;   // target: global reference, 1 / sum
  float Md, invSd;   // draft
  float sig;         // sigma of the current residual (R = sig R~; 1 / S_t before any map)
  SpecConst sc;      // SpecInfer instance: the residual's threshold K and exponent constants
  const float (*tab)[2];  // SpecInfer instance: 2^(j/64) as double-floats
};

// 2^(z c - M): p~ or q~ of one element from its raw logit.
__device__ __forceinline__ float exp_of(float z, float c, float M) {
  return ex2(__fmaf_rn(z, c, -M));
}

// The unnormalised ResiSpec residual R~ after the first nm maps,
// element-wise (no rejected-token zeroing: the caller applies it): the
// GetProxy residual r = min(Z q, R) + lambda (R - min(Z q, R)),
// R' = r / sum r, in the units above.  The map's two parts from R~ and q~:
// m = min(k q~, R~) and the capacity R~ - m.  (SpecInfer keeps no maps: its
// residual is one threshold away from p, see specinfer.cuh.)
__device__ __forceinline__ float2 min_part2(float2 k, float2 q, float2 R) {
  const float2 kq = __fmul2_rn(k, q);
  return make_float2(fminf(kq.x, R.x), fminf(kq.y, R.y));
}

// Kinds of residual chain: SpecInfer (the threshold of specinfer.cuh, its
// own kernel instance); ResiSpec maps with the draft q as the test
// denominator D throughout (Algorithm 1); ResiSpec maps with the
// proxy as the next denominator (the paper's EAGLE integration, App. C).
// With the proxy update the map is written with the current denominator:
// m = min(k D~, R~), t = R~ - m, R~' = m + lambda t, and the proxy off the
// rejected token is K = R - r = (1 - lambda) t, so D~' = t in units of
// sigma_before (1 - lambda): one more value per element, no more work.
enum : int { kChainSpec = 0, kChainResi = 1, kChainResiDenom = 2 };

// The chain on one element: R~ and the denominator D~ (a draft value q~ on
// entry; changed only by kChainResiDenom).  No rejected-token rule is
// applied here (the callers do).
template <int KIND>
__device__ __forceinline__ float apply_chain(const StreamHead& S2, int nm, float R, float& D) {
  for (int i = 0; i < nm; ++i) {
    const float2 mp = S2.map[i];
    const float m = fminf(__fmul_rn(mp.x, D), R);
    const float t = __fmaf_rn(m, -1.f, R);
    R = __fmaf_rn(mp.y, t, m);
    if constexpr (KIND == kChainResiDenom) D = t;
  }
  return R;
}

// The same on pairs: every lane rounds exactly like apply_chain.
template <int NP, int KIND>
__device__ __forceinline__ void apply_chain_pairs(const StreamHead& S2, int nm, float2 (&R)[NP],
                                                  float2 (&D)[NP]) {
  for (int i = 0; i < nm; ++i) {
    const float2 mp = S2.map[i];
    const float2 k = dup2(mp.x);
    const float2 lam = dup2(mp.y);
#pragma unroll
    for (int j = 0; j < NP; ++j) {
      const float2 m = min_part2(k, D[j], R[j]);
      const float2 t = __ffma2_rn(m, dup2(-1.f), R[j]);
      R[j] = __ffma2_rn(lam, t, m);
      if constexpr (KIND == kChainResiDenom) D[j] = t;
    }
  }
}

template <int NP>
__device__ __forceinline__ void apply_chain_any(const StreamHead& S2, int chain, int nm,
                                                float2 (&R)[NP], float2 (&D)[NP]) {
  if (chain == kChainResiDenom) apply_chain_pairs<NP, kChainResiDenom>(S2, nm, R, D);
  else apply_chain_pairs<NP, kChainResi>(S2, nm, R, D);
}

// Zero the residual at rejected tokens (ResiSpec: r(x0) = 0 and the later
// maps keep a zero at zero) in the vector whose first token is `base`.
template <int VEC>
__device__ __forceinline__ void zero_rejected_vec(const StreamHead& S2, int nm, int base,
                                                  float (&R)[VEC]) {
  for (int i = 0; i < nm; ++i) {
    const unsigned d = (unsigned)(S2.rej[i] - base);
#pragma unroll
    for (int j = 0; j < VEC; ++j)
      if ((unsigned)j == d) R[j] = 0.f;
  }
}

// Final values (the distribution being sampled) of vector g of a ring
// stage row (g = h THREADS + t is vector h of thread t's chunk): p when no
// map is pending, else the residual, R = sig R~ (zero at the rejected
// tokens).  base: its first token.
template <int THREADS, bool BF16, bool SPEC>
__device__ __forceinline__ void final_values(const StreamHead& S2, const VisitScalars& K,
                                             int chain, int nm, int base,
                                             const unsigned char* rt, const unsigned char* rd,
                                             int g, float (&v)[BF16 ? 8 : 4]) {
  constexpr int VEC = BF16 ? 8 : 4;
  constexpr int NP = VEC / 2;
  float z[VEC];
  unpack_vec<BF16>(reinterpret_cast<const uint4*>(rt)[g], z);
  if constexpr (SPEC) {
    if (nm > 0) {  // SpecInfer residual (p~ - K q~)_+ / T (specinfer.cuh)
      float zd[VEC];
      unpack_vec<BF16>(reinterpret_cast<const uint4*>(rd)[g], zd);
#pragma unroll
      for (int j = 0; j < VEC; ++j)
        v[j] = __fmul_rn(df_value(spec_residual(z[j], zd[j], K.sc, K.tab)), K.sig);
      return;
    }
  }
  const float2 c2 = dup2(K.c);
  float2 R[NP];
#pragma unroll
  for (int j = 0; j < NP; ++j)
    R[j] = ex2x2(__ffma2_rn(make_float2(z[2 * j], z[2 * j + 1]), c2, dup2(-K.Mt)));
  if (nm == 0) {
#pragma unroll
    for (int j = 0; j < NP; ++j) {
      const float2 r = __fmul2_rn(R[j], dup2(K.invSt));
      v[2 * j] = r.x;
      v[2 * j + 1] = r.y;
    }
    return;
  }
  unpack_vec<BF16>(reinterpret_cast<const uint4*>(rd)[g], z);
  float2 q[NP];
#pragma unroll
  for (int j = 0; j < NP; ++j)
    q[j] = ex2x2(__ffma2_rn(make_float2(z[2 * j], z[2 * j + 1]), c2, dup2(-K.Md)));
  apply_chain_any<NP>(S2, chain, nm, R, q);
#pragma unroll
  for (int j = 0; j < NP; ++j) {
    const float2 r = __fmul2_rn(R[j], dup2(K.sig));
    v[2 * j] = r.x;
    v[2 * j + 1] = r.y;
  }
  zero_rejected_vec<VEC>(S2, nm, base, v);
}

// ---------------------------------------------------------------- sampler
// Inverse-CDF draw inside one CTA: the smallest slice offset whose inclusive
// mass prefix exceeds `tau` (mass units 2^-44).
//   1. One pass over the slice sums the values of every warp's share of a
//      chunk (fp32, a fixed butterfly order) and adds it, rounded to the
//      fixed-point unit, into the chunk's total with one shared-memory
//      atomic per warp and chunk (integer sums: the totals do not depend on
//      the order of the atomics; no barrier inside the pass).  `ck` holds
//      one total per chunk.
//   2. One warp scans the chunk totals and finds the chunk that holds tau.
//   3. That chunk's vectors are read again; a block-wide scan of their exact
//      fixed-point masses in token order (vector h of thread t is token block
//      h THREADS + t) finds the vector, and its thread walks its values.
// The chunk totals carry the fp32 rounding of step 1 (about 1e-7 of the
// mass), so they can place tau in a neighbouring chunk only when it lies
// that close to a chunk boundary; if tau then falls past the chunk's exact
// total (or rounding leaves it past the slice's total), the last token with
// positive mass is taken.  Returns the token's offset in the slice (-1 if the
// slice has no mass).
constexpr int kMaxSearchChunks = 128;

// Step 1 of a search: the slice's chunk totals ck[k] (fixed point), from
// the records of the pass that defined the distribution, or from a pass.
template <int THREADS, bool BF16, bool SPEC>
__device__ void search_totals(const StreamHead& S2, unsigned long long* ck, unsigned char* ring,
                              const Src& s, const VisitScalars& K, int chain, int lo,
                              const ChunkRec& cr) {
  using G = StreamGeom<THREADS, BF16>;
  constexpr int VEC = G::VEC;
  constexpr int NW = THREADS / 32;
  const int lane = threadIdx.x & 31;
  const int nm = S2.nmaps;
  const int NK = (s.nloc + G::CE - 1) / G::CE;  // <= kMaxSearchChunks (slices <= 2^18)
  for (int k = threadIdx.x; k < NK; k += THREADS) ck[k] = 0ull;
  __syncthreads();
  if (cr.kind != 0) {
    // chunk totals from the records of the pass that defined the distribution
    for (int k = threadIdx.x; k < NK; k += THREADS) {
      float m = 0.f;
      for (int w = 0; w < NW; ++w) {
        const float r0 = S2.crec[0][k * NW + w], r1 = S2.crec[1][k * NW + w];
        float v;
        if (cr.kind == 1) v = __fmul_rn(__fmul_rn(r1, ex2(__fsub_rn(r0, cr.a))), cr.b);
        else if (cr.kind == 2) v = __fmul_rn(__fmaf_rn(cr.a, r1, r0), cr.b);
        else v = __fmul_rn(r0, cr.b);
        m = __fadd_rn(m, v);
      }
      ck[k] = to_fix(m);
    }
  } else stream_pass<THREADS, BF16>(ring, s, [&](const unsigned char* rt,
                                                         const unsigned char* rd, int k) -> bool {
    float2 acc2 = make_float2(0.f, 0.f);
#pragma unroll
    for (int h = 0; h < G::VPT; ++h) {
      float v[VEC];
      final_values<THREADS, BF16, SPEC>(S2, K, chain, nm,
                                        lo + k * G::CE + (h * THREADS + (int)threadIdx.x) * VEC,
                                        rt, rd, h * THREADS + (int)threadIdx.x, v);
#pragma unroll
      for (int j = 0; j < VEC / 2; ++j) acc2 = __fadd2_rn(acc2, make_float2(v[2 * j], v[2 * j + 1]));
    }
    const float acc = group_sum<5>(__fadd_rn(acc2.x, acc2.y));
    if (lane == 0) {
      const unsigned long long a = to_fix(acc);
      if (a) atomicAdd(ck + k, a);
    }
    return false;
  });
  __syncthreads();
}

// Step 2 (warp 0): the chunk holding tau in the inclusive prefix of ck, and
// tau's remainder inside it; a threshold past the slice's total takes its
// last chunk with mass (force).  Returns the chunk (-1: no mass).
__device__ __forceinline__ int search_chunk_of(const unsigned long long* ck, int NK,
                                               unsigned long long tau, bool& force,
                                               unsigned long long& rem) {
  const int lane = threadIdx.x & 31;
  unsigned long long run = 0;
  int kfound = -1, klast = -1;
  unsigned long long before = 0;
  for (int base = 0; base < NK; base += 32) {
    const int k = base + lane;
    const unsigned long long m = k < NK ? ck[k] : 0ull;
    unsigned long long incl = m;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    incl += run;
    const unsigned cross = __ballot_sync(0xffffffffu, k < NK && incl > tau);
    const unsigned pos = __ballot_sync(0xffffffffu, m > 0);
    if (pos) klast = base + 31 - __clz(pos);
    if (kfound < 0 && cross) {
      const int l = __ffs(cross) - 1;
      kfound = base + l;
      before = __shfl_sync(0xffffffffu, incl - m, l);
    }
    run = __shfl_sync(0xffffffffu, incl, 31);
  }
  force = kfound < 0;
  rem = kfound >= 0 ? tau - before : 0ull;
  return kfound >= 0 ? kfound : klast;
}

// Step 3: the token of chunk ks (this thread's vectors at stage stg) whose
// exact prefix mass crosses t, or with force (or when no vector holds t) the
// chunk's last token with mass.  Returns its offset in the slice.  H.misc[4]
// and H.misc[7] hold -1 on entry (set before a barrier).
template <int THREADS, bool BF16, bool SPEC>
__device__ int search_in_chunk(Head& H, const StreamHead& S2, const unsigned char* stg,
                               const Src& s, const VisitScalars& K, int chain, int lo, int ks,
                               bool force, unsigned long long t) {
  using G = StreamGeom<THREADS, BF16>;
  constexpr int VEC = G::VEC;
  constexpr int NW = THREADS / 32;
  static_assert(G::VPT * NW <= 32, "one scan lane per warp segment");
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nm = S2.nmaps;
  float v[G::VPT][VEC];
  unsigned long long mv[G::VPT], ex[G::VPT];
  int lastpos = -1;
#pragma unroll
  for (int h = 0; h < G::VPT; ++h) {
    const int g = h * THREADS + (int)threadIdx.x;
    final_values<THREADS, BF16, SPEC>(S2, K, chain, nm, lo + ks * G::CE + g * VEC, stg,
                                      stg + G::RB, g, v[h]);
    mv[h] = 0;
#pragma unroll
    for (int j = 0; j < VEC; ++j) {
      mv[h] += to_fix(v[h][j]);
      if (v[h][j] > 0.f && ks * G::CE + g * VEC + j < s.nloc) lastpos = g * VEC + j;
    }
    unsigned long long incl = mv[h];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    ex[h] = incl - mv[h];
    if (lane == 31) H.seg[h * NW + warp] = incl;
  }
  __syncthreads();
  if (warp == 0) {  // exclusive prefix of the warp segments in token order
    const unsigned long long m = lane < G::VPT * NW ? H.seg[lane] : 0ull;
    unsigned long long incl = m;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    __syncwarp();
    if (lane < G::VPT * NW) H.seg[lane] = incl - m;
  }
  __syncthreads();
  if (lastpos >= 0) atomicMax(&H.misc[7], lastpos);  // the chunk's last token with mass
  if (!force) {
#pragma unroll
    for (int h = 0; h < G::VPT; ++h) {
      const unsigned long long a0 = H.seg[h * NW + warp] + ex[h];
      if (mv[h] > 0 && a0 <= t && t < a0 + mv[h]) {
        unsigned long long a = a0;
        int pick = (h * THREADS + (int)threadIdx.x) * VEC + VEC - 1;
#pragma unroll
        for (int j = 0; j < VEC; ++j) {
          a += to_fix(v[h][j]);
          if (a > t) { pick = (h * THREADS + (int)threadIdx.x) * VEC + j; break; }
        }
        H.misc[4] = pick;
      }
    }
  }
  __syncthreads();
  // no vector holds tau (forced, or tau past the chunk's exact total): the
  // chunk's last token with positive mass
  const int pick = H.misc[4] >= 0 ? H.misc[4] : H.misc[7];
  __syncthreads();
  return pick < 0 ? -1 : ks * G::CE + pick;
}


// Step 3 for one warp, for a row's own distribution (no residual map: the
// drafting step's draws from q): the token search_in_chunk finds, found by
// one warp alone over the whole chunk (every vector landed and visible to
// the warp).  The values are final_values' without a map, bit for bit:
// 2^(z c - M) / S.  The warp walks the chunk's vectors in token order, 32 at a
// time (lane l takes vector 32 i + l: conflict-free loads), with an exact
// 64-bit scan of their fixed-point totals on top of the groups before; the
// lane whose vector holds t walks its values.  Integer sums are exact, so
// the crossing token is the one a block-wide scan finds.
template <int THREADS, bool BF16>
__device__ int warp_draw_in_chunk(const unsigned char* stg, int nloc, float c, float M, float inv,
                                  int ks, bool force, unsigned long long t) {
  using G = StreamGeom<THREADS, BF16>;
  constexpr int VEC = G::VEC;
  constexpr int PV = G::VPT * THREADS / 32;  // vectors per lane
  const int lane = threadIdx.x & 31;
  auto values = [&](int g, float (&v)[VEC]) {
    float z[VEC];
    unpack_vec<BF16>(reinterpret_cast<const uint4*>(stg)[g], z);
#pragma unroll
    for (int j = 0; j < VEC; ++j) v[j] = __fmul_rn(ex2(__fmaf_rn(z[j], c, -M)), inv);
  };
  int pick = -1;
  if (!force) {
    unsigned long long run = 0;  // mass of the groups before
#pragma unroll 1
    for (int i = 0; i < PV; ++i) {
      const int g = i * 32 + lane;
      float v[VEC];
      values(g, v);
      unsigned long long m = 0;
#pragma unroll
      for (int j = 0; j < VEC; ++j) m += to_fix(v[j]);
      unsigned long long incl = m;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long n = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += n;
      }
      incl += run;
      const unsigned long long a0 = incl - m;
      const unsigned hit = __ballot_sync(0xffffffffu, m > 0 && a0 <= t && t < incl);
      if (hit) {
        const int l = __ffs(hit) - 1;
        if (lane == l) {
          unsigned long long a = a0;
          pick = g * VEC + VEC - 1;
#pragma unroll
          for (int j = 0; j < VEC; ++j) {
            a += to_fix(v[j]);
            if (a > t) { pick = g * VEC + j; break; }
          }
        }
        pick = __shfl_sync(0xffffffffu, pick, l);
        break;
      }
      run = __shfl_sync(0xffffffffu, incl, 31);
    }
  }
  if (pick < 0) {  // forced, or t past the chunk's total: its last token with mass
    int last = -1;
#pragma unroll 1
    for (int i = 0; i < PV; ++i) {
      const int g = i * 32 + lane;
      float v[VEC];
      values(g, v);
#pragma unroll
      for (int j = 0; j < VEC; ++j)
        if (v[j] > 0.f && ks * G::CE + g * VEC + j < nloc) last = g * VEC + j;
    }
    pick = __reduce_max_sync(0xffffffffu, last);
  }
  return pick < 0 ? -1 : ks * G::CE + pick;
}

template <int THREADS, bool BF16, bool SPEC>
__device__ int stream_search(Head& H, const StreamHead& S2, unsigned long long* ck,
                             unsigned char* ring, const Src& s, const VisitScalars& K, int chain,
                             int lo, unsigned long long tau, const ChunkRec& cr) {
  using G = StreamGeom<THREADS, BF16>;
  const int NK = (s.nloc + G::CE - 1) / G::CE;
  search_totals<THREADS, BF16, SPEC>(S2, ck, ring, s, K, chain, lo, cr);
  if ((threadIdx.x >> 5) == 0) {
    bool force;
    unsigned long long rem;
    const int k = search_chunk_of(ck, NK, tau, force, rem);
    if (threadIdx.x == 0) {
      H.misc[0] = k;
      H.misc[3] = force;
      H.fixd[0] = rem;
      H.misc[4] = -1;
      H.misc[7] = -1;
    }
  }
  __syncthreads();
  const int ks = H.misc[0];
  if (ks < 0) return -1;
  const bool force = H.misc[3] != 0;
  const unsigned long long t = H.fixd[0];
  // the chosen chunk's values (this thread's vectors: held in the ring, or
  // copied again into ring stage 0, which only this thread's copies write)
  const unsigned char* stg = ring;
  if (s.held) {
    stg = held_stage<THREADS, BF16>(ring, s, ks);
  } else {
    copy_chunk<THREADS, BF16>(s, ks, ring, s.rows == 2);
    cp_async_wait<0>();
  }
  return search_in_chunk<THREADS, BF16, SPEC>(H, S2, stg, s, K, chain, lo, ks, force, t);
}

// Final draw of a visit: every CTA picks the CTA whose mass range holds
// u * total (as the resident kernel's sampler); that CTA searches its slice.
template <int THREADS, bool BF16, bool SPEC>
__device__ bool stream_sample(Head& H, StreamHead& S2, unsigned char* ring, const VerifyParams& P,
                              const Src& s_in, const VisitScalars& K, int chain, int mass_kind,
                              const Pending& Pm, float u, int b, int depth, int lo,
                              uint32_t rank, uint32_t C, int& xp, uint32_t& xph, bool& timeout,
                              const ChunkRec& cr) {
  using G = StreamGeom<THREADS, BF16>;
  constexpr int VEC = G::VEC;
  constexpr int NW = THREADS / 32;
  const int nm = S2.nmaps;
  // the visit's rows, in the ring layout they were loaded with (a residual
  // left unchanged by degenerate rejections still streams both rows)
  const Src& s = s_in;
  if (P.out_dist || mass_kind == 0) {
    // every CTA: values of its slice (written out when asked) and their sum
    float* dist = P.out_dist ? P.out_dist + (size_t)b * P.V + lo : nullptr;
    float sum = 0.f;
    stream_pass<THREADS, BF16>(ring, s, [&](const unsigned char* rt,
                                                    const unsigned char* rd, int k) -> bool {
#pragma unroll
      for (int h = 0; h < G::VPT; ++h) {
        float v[VEC];
        const int e0 = k * G::CE + (h * THREADS + (int)threadIdx.x) * VEC;  // offset in the slice
        final_values<THREADS, BF16, SPEC>(S2, K, chain, nm, lo + e0, rt, rd,
                                          h * THREADS + (int)threadIdx.x, v);
#pragma unroll
        for (int j = 0; j < VEC; ++j) {
          sum += v[j];
          if (dist && e0 + j < s.nloc) dist[e0 + j] = v[j];
        }
      }
      return false;
    });
    if (mass_kind == 0) {
      float o[8];
      int of;
      exchange<NW, false>(H, sum, 0.f, 0.f, 0.f, 0, -1, xp, xph, rank, C, o, of);
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
  // chunk totals of the search: the children's logit slots, unused by the draw
  const int pick = stream_search<THREADS, BF16, SPEC>(
      H, S2, reinterpret_cast<unsigned long long*>(S2.kzt), ring, s, K, chain, lo, tau, cr);
  if (threadIdx.x == 0) P.out_tokens[(size_t)b * (P.D + 1) + depth] = lo + max(pick, 0);
  return true;
}

// Cluster total of N double-float partials per thread (SpecInfer sums):
// each CTA reduces its threads' values in a fixed order (warp butterflies,
// then one warp over the warps' values), pushes the CTA's value through the
// exchange (only thread 0 contributes, so the exchange's own fp32 sums add
// zeros), and every CTA adds the received per-CTA values in rank order, so
// that all CTAs obtain the same bits.
template <int NW, int N>
__device__ __forceinline__ bool df_exchange(Head& H, DF (&v)[N], DF (&tot)[N], int& xp,
                                            uint32_t& xph, uint32_t rank, uint32_t C) {
  static_assert(N <= 2 && N * NW <= 32, "two double-floats per warp in the segment slots");
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  DF* wdf = reinterpret_cast<DF*>(H.seg);
#pragma unroll
  for (int i = 0; i < N; ++i) {
    v[i] = df_group_sum<5>(v[i]);
    if (lane == 0) wdf[i * NW + warp] = v[i];
  }
  __syncthreads();
  float a[4] = {0.f, 0.f, 0.f, 0.f};
  if (warp == 0) {
#pragma unroll
    for (int i = 0; i < N; ++i) {
      const DF c = df_group_sum<4>(lane < NW ? wdf[i * NW + lane] : df(0.f));
      if (lane == 0) {
        a[2 * i] = c.hi;
        a[2 * i + 1] = c.lo;
      }
    }
  }
  float o[8];
  int oflags;
  exchange<NW, false, 2 * N>(H, a[0], a[1], a[2], a[3], 0, -1, xp, xph, rank, C, o, oflags);
#pragma unroll
  for (int i = 0; i < N; ++i) {
    tot[i] = df(0.f);
    for (uint32_t r = 0; r < C; ++r)
      tot[i] = df_add(tot[i], DF{H.part[r][2 * i], H.part[r][2 * i + 1]});
  }
  return !(oflags & kFlagTimeout);
}

// ---------------------------------------------------------------- kernel
// VAR: the instance that carries the optional paths (Z_applied, proxy
// denominator, level fill, drafting, phase counters).  The default instance
// compiles them out: their code, even untaken, costs the hot loops
// instruction-cache misses.
template <int THREADS, bool BF16, bool VAR, bool SPEC>
__global__ void __launch_bounds__(THREADS, THREADS >= 512 ? 2 : 4)
    stream_kernel(const __grid_constant__ VerifyParams P) {
  using G = StreamGeom<THREADS, BF16>;
  constexpr int NW = THREADS / 32;
  constexpr int VEC = G::VEC;
  constexpr int es = BF16 ? 2 : 4;
  extern __shared__ __align__(128) unsigned char smem[];
  Head& H = *reinterpret_cast<Head*>(smem);
  StreamHead& S2 = *reinterpret_cast<StreamHead*>(smem + kHeadBytes);
  unsigned char* ring = smem + kHeadBytes + kStreamHeadBytes;  // S stages of SB bytes
  int16_t* par = reinterpret_cast<int16_t*>(ring + G::RING);
  int16_t* first_child = par + P.npad;
  int16_t* next_sib = first_child + P.npad + 16;
  int32_t* cand_s = reinterpret_cast<int32_t*>(next_sib + P.npad);

  // Nothing is read before the preceding work on the stream has completed;
  // the next launch may be scheduled from here on (it waits the same way).
  grid_dependency_wait();
  grid_launch_dependents();
  const int tid = threadIdx.x;
  const uint32_t rank = cluster_ctarank();
  const uint32_t C = cluster_nctarank();
  const int b = (int)cluster_id_x();
  const int N = P.N, V = P.V, D = P.D;
  const int L = P.slice;
  const int lo = (int)rank * L;
  const int nloc = max(0, min(V, lo + L) - lo);
  // SPEC: the SpecInfer instance (Eq. 2, evaluated as in specinfer.cuh);
  // the others run ResiSpec (Algorithm 1)
  const int chain = SPEC ? kChainSpec : ((VAR && P.denom_update) ? kChainResiDenom : kChainResi);
  const bool drafting = VAR && P.draft_out != nullptr;
  const bool bf16 = BF16;

  int err = 0;
  int info = 0;
  int depth = 0, rejects = 0;
  int node = -1, row = 0;
  uint32_t xph = 0;
  int xp = 0;
  const int lane = tid & 31, warp = tid >> 5;
  // chunk records for the final draw (ChunkRec; not in the instance with the
  // optional paths)
  const bool rec_ok = !VAR && ((nloc + G::CE - 1) / G::CE) * NW <= kMaxChunkRecs;
  // drafting: the normaliser records the draft row's chunk masses, from
  // which every child's draw finds its chunk (ChunkRec kind 1 on q)
  const bool rec_draft = VAR && P.draft_out != nullptr &&
                         ((nloc + G::CE - 1) / G::CE) * NW <= kMaxChunkRecs;

  // Kernel setup: exchange barriers, the tree's child lists and the
  // candidates.  It runs while the first chunks of the root's rows are in
  // flight (the root has children exactly when N > 0 in a valid tree, since
  // node 0's parent can only be the root).
  auto setup = [&] {
    if (tid < 4) H.pubv[tid] = 0.f;
    if constexpr (SPEC)  // the 2^(j/64) table, read at lane-dependent indices
      for (int i = tid; i < 2 * kExp2Tab; i += THREADS) (&S2.tab[0][0])[i] = (&P.exp2_tab[0][0])[i];
    if (tid == 0) {
      mbar_init(smem_addr(&H.xbar[0]), 1);
      mbar_init(smem_addr(&H.xbar[1]), 1);
      fence_mbar_init();
    }
    for (int i = tid; i < P.npad + 16; i += THREADS) first_child[i] = -1;
    int bad = 0;
    for (int i = tid; i < N; i += THREADS) {
      const int p = __ldg(P.parents + (size_t)b * P.parents_stride + i);
      const bool ok = p >= -1 && p < i;
      bad |= !ok;
      par[i] = (int16_t)(ok ? p : -2);
      cand_s[i] = drafting ? -1 : __ldg(P.cand + (size_t)b * N + i);
      if (drafting && rank == 0) P.draft_out[(size_t)b * N + i] = -1;
    }
    const bool tree_bad = __syncthreads_or(bad) != 0;
    build_children(par, first_child, next_sib, N);
    __syncthreads();
    cluster_sync();  // every peer has started: its receive slots may now be written
    if (tree_bad) err = kErrTree;
  };

  // Drafting (Algorithm 1's "x_1..x_k ~ Q i.i.d."): the children of each
  // visited node are drawn here from the node's tempered draft row, after
  // its normaliser, instead of being read from cand.
  auto draft_children = [&](int c1d, const VisitScalars& K, size_t rbase) {
    // per-CTA draft masses from the normaliser exchange, the CTA and the
    // threshold inside it of each child's draw; kept in the children's logit
    // slots (refilled below) and the rejected-token list (empty until the
    // node's first map), which the searches do not touch
    static_assert(offsetof(StreamHead, kzd) == offsetof(StreamHead, kzt) + sizeof(StreamHead::kzt) &&
                      offsetof(StreamHead, kzt) % 8 == 0 &&
                      sizeof(StreamHead::kzt) + sizeof(StreamHead::kzd) >=
                          kMaxKids * sizeof(unsigned long long),
                  "draft thresholds fit the logit slots");
    unsigned long long* tau = reinterpret_cast<unsigned long long*>(S2.kzt);
    int* owner = S2.rej;
    // per-CTA draft masses (fixed point), in the sampler's segment slots
    static_assert(sizeof(Head::seg) >= kMaxCluster * sizeof(unsigned long long),
                  "per-CTA masses fit the segment slots");
    unsigned long long* cmass = H.seg;
    if (tid < (int)C) cmass[tid] = to_fix(__fmul_rn(H.part[tid][3], ref_scale(H.part[tid][2], K.Md, K.invSd)));
    if (tid == 0) {
      int i = 0;
      for (int cn = c1d; cn >= 0 && i < kMaxKids; cn = next_sib[cn]) ++i;
      H.misc[6] = i;
    }
    __syncthreads();
    const int nk = H.misc[6];
    if (tid < nk) {  // child tid's draw: its CTA and the threshold inside it
      int cn = c1d;
      for (int k = 0; k < tid; ++k) cn = next_sib[cn];
      unsigned long long total = 0;
      for (uint32_t r = 0; r < C; ++r) total += cmass[r];
      const unsigned long long kk = tau[tid];  // the draw's 24 bits (normaliser pass)
      const unsigned long long t = (__umul64hi(kk, total) << 40) | ((kk * total) >> 24);
      unsigned long long a = 0;
      int r_own = total > 0 ? (int)C - 1 : -1;
      for (uint32_t r = 0; r < C && total > 0; ++r) {
        const unsigned long long m = cmass[r];
        if (a + m > t) { r_own = (int)r; break; }
        a += m;
      }
      tau[tid] = t > a ? t - a : 0ull;
      owner[tid] = r_own;
    }
    __syncthreads();
    // q values come out of the sampler's search with the draft row in
    // place of the target row and the draft's scalars
    Src sq;
    sq.t = static_cast<const char*>(P.zd) + (rbase + (size_t)lo) * es;
    sq.d = sq.t;
    sq.rows = 1;
    sq.nloc = nloc;
    sq.vec = P.use_tma != 0;
    sq.held = false;
    VisitScalars Kq = K;
    Kq.Mt = K.Md;
    Kq.invSt = K.invSd;
    // The children this CTA owns: the draft row's chunk totals once (from
    // the normaliser's records, or one pass), each child's chunk and the
    // remainder of its threshold (one warp per child), then the owned
    // children's chunks copied together, one single-row ring stage each, and
    // one in-chunk search per child, one warp per child (the steps of
    // stream_search, shared across the children).  Chunk totals in the
    // residual maps' slots (no map exists before the node's accept tests),
    // each child's chunk in the rejected-child slots.
    static_assert(sizeof(StreamHead::map) >= kMaxSearchChunks * sizeof(unsigned long long),
                  "search chunk totals fit the map slots");
    unsigned long long* ck = reinterpret_cast<unsigned long long*>(S2.map);
    int16_t* kchunk = S2.rejk;  // -2: not owned; -1: no mass; else chunk | force << 13
    bool mine = false;
    for (int i = 0; i < nk; ++i) mine |= owner[i] == (int)rank;
    if (mine) {
      search_totals<THREADS, BF16, SPEC>(S2, ck, ring, sq, Kq, chain, lo,
                                         ChunkRec{rec_draft ? 1 : 0, K.Md, K.invSd});
      const int NK = (nloc + G::CE - 1) / G::CE;
      for (int i = warp; i < nk; i += NW) {
        int16_t code = -2;
        if (owner[i] == (int)rank) {
          bool force;
          unsigned long long rem;
          const int kc = search_chunk_of(ck, NK, tau[i], force, rem);
          if (lane == 0) tau[i] = rem;
          code = (int16_t)(kc < 0 ? -1 : kc | (force ? 1 << 13 : 0));
        }
        if (lane == 0) kchunk[i] = code;
      }
      __syncthreads();
      // batches of up to min(ring stages, warps) children with mass
      const int width = min(ring_depth<THREADS, BF16>(false), NW);
      for (int i0 = 0, cn0 = c1d; i0 < nk;) {
        int i1 = i0, n = 0;
        for (; i1 < nk && n < width; ++i1)
          if (kchunk[i1] >= 0)
            copy_chunk<THREADS, BF16>(sq, kchunk[i1] & 0x1fff, ring + (n++) * G::RB, false);
        cp_async_wait<0>();
        __syncthreads();  // every thread's vectors of the batch's chunks have landed
        // up to two children: each searched by the whole CTA (a block-wide
        // scan); more: one warp per child, all at once
        const bool by_warp = n > 2;
        for (int i = i0, j = 0, cn = cn0; i < i1; ++i, cn = next_sib[cn]) {
          if (kchunk[i] == -2) continue;
          const int kc = kchunk[i] & 0x1fff;
          const bool force = (kchunk[i] >> 13) != 0;
          if (kchunk[i] < 0) {
            if (tid == 0) P.draft_out[(size_t)b * N + cn] = lo;
          } else if (by_warp) {
            if (j++ != warp) continue;
            const int pick = warp_draw_in_chunk<THREADS, BF16>(ring + warp * G::RB, nloc, K.c,
                                                               K.Md, K.invSd, kc, force, tau[i]);
            if (lane == 0) P.draft_out[(size_t)b * N + cn] = lo + max(pick, 0);
          } else {
            if (tid == 0) {
              H.misc[4] = -1;
              H.misc[7] = -1;
            }
            __syncthreads();
            const int pick = search_in_chunk<THREADS, BF16, SPEC>(
                H, S2, ring + (j++) * G::RB, sq, Kq, chain, lo, kc, force, tau[i]);
            if (tid == 0) P.draft_out[(size_t)b * N + cn] = lo + max(pick, 0);
          }
        }
        __syncthreads();  // the stages are reused by the next batch
        for (int i = i0; i < i1; ++i) cn0 = next_sib[cn0];
        i0 = i1;
      }
    }
    cluster_sync();  // every drawn token written (release / acquire at cluster scope)
    // the children's tokens and their raw logits
    if (tid < nk) {
      int cn = c1d;
      for (int k = 0; k < tid; ++k) cn = next_sib[cn];
      const int x = __ldcg(P.draft_out + (size_t)b * N + cn);
      cand_s[cn] = x;
      const bool okx = x >= 0 && x < V;
      S2.kzt[tid] = okx ? raw_logit(P.zt, rbase + (size_t)x, bf16) : 0.f;
      S2.kzd[tid] = okx ? raw_logit(P.zd, rbase + (size_t)x, bf16) : 0.f;
    }
    __syncthreads();
  };

  // optional phase counters (thread 0 of every CTA; rank 0 writes them)
  const bool prof = VAR && P.out_phase != nullptr;
  auto mark = [&](int ph) {
    if (prof && tid == 0) {
      const unsigned long long now = clock64();
      S2.phc[S2.ph_cur] += now - S2.ph_last;
      S2.ph_last = now;
      S2.ph_cur = ph;
    }
  };
  if (prof && tid == 0) {
    for (int k = 0; k < kPhases; ++k) S2.phc[k] = 0ull;
    S2.ph_last = clock64();
    S2.ph_cur = kPhaseSetup;
  }

  for (bool first = true; !err; first = false) {
    int c1 = first ? -1 : first_child[node + 1];
    const bool need_draft = first ? N > 0 : c1 >= 0;
    const size_t rbase = (size_t)b * P.seq_stride + (size_t)row * V;
    Src src;
    src.t = static_cast<const char*>(P.zt) + (rbase + (size_t)lo) * es;
    src.d = static_cast<const char*>(P.zd) + (rbase + (size_t)lo) * es;
    src.rows = need_draft ? 2 : 1;
    src.nloc = nloc;
    src.vec = P.use_tma != 0;
    src.held = false;

    // Per-visit state in S2 is written by every thread with identical
    // values (each thread reads back its own writes), so no barrier is
    // needed to publish it; the barrier at the end of the previous visit
    // orders these writes after every read of the old values.
    S2.nmaps = 0;

    mark(kPhaseNorm);
    // ---- tempered normaliser (S2): online (reference, sum) per row; while
    // the first chunks are in flight, one thread per child reads its token's
    // raw logits and draws its accept uniform (one Philox block per logit
    // row r: word 0 is the accept draw of node r - 1, word 1 the final draw
    // at row r), and one more thread draws the visit's final uniform
    float mt = kNoRef, md = kNoRef;
    float2 st2 = make_float2(0.f, 0.f), sd2 = make_float2(0.f, 0.f);
    float dmin = INFINITY;  // Z_applied: smallest z_t - z_d of the slice
    ChunkRec crec{0, 0.f, 0.f};  // records of this visit's final distribution
    const bool zapp = VAR && !SPEC && P.z_applied != 0;
    // (child t is found by walking t siblings; the loaded logits stay in
    // registers until the pass ends, so no warp waits for them; the draws
    // are computed by the last threads)
    auto nth_child = [&](int t) {
      int cn = c1;
      for (int k = 0; k < t && cn >= 0; ++k) cn = next_sib[cn];
      return cn;
    };
    bool have_kid = false;
    float kz_t = 0.f, kz_d = 0.f;
    stream_pass_pre<THREADS, BF16>(ring, src,
        [&] {
          if (first) {
            setup();
            c1 = first_child[0];
          }
          if (tid < kMaxKids && need_draft && !err && !drafting) {
            const int cn = nth_child(tid);
            if (cn >= 0) {
              const int x = cand_s[cn];
              const bool okx = x >= 0 && x < V;
              have_kid = true;
              kz_t = okx ? raw_logit(P.zt, rbase + (size_t)x, bf16) : 0.f;
              kz_d = okx ? raw_logit(P.zd, rbase + (size_t)x, bf16) : 0.f;
            }
          }
          const int j = THREADS - 1 - tid;  // kMaxKids < THREADS - kMaxKids
          if (j < kMaxKids && need_draft && !err) {
            const int cn = nth_child(j);
            if (cn >= 0) {
              // U(seed, b, cn + 1, .): word 0 the accept draw; word 2 the
              // drafting draw, kept as its 24-bit integer in the child's
              // threshold slot (draft_children)
              const U64x4 r = philox4x64_10((uint64_t)(cn + 1), (uint64_t)b, 0, 0, P.seed, 0);
              S2.kua[j] = u24(r.w[0]);
              if (drafting)
                reinterpret_cast<unsigned long long*>(S2.kzt)[j] =
                    (unsigned long long)(u24(r.w[2]) * 16777216.f);
            }
          } else if (j == kMaxKids) {
            S2.ufin = uniform_draw(P.seed, (uint32_t)b, (uint32_t)row, 1);
          }
        },
        [&](const unsigned char* rt, const unsigned char* rd, int k) -> bool {
          if (err) return true;  // invalid tree (uniform over the cluster)
          float2 zt[G::NP], zd[G::NP];
          load_pairs<THREADS, BF16>(rt, zt);
          if (need_draft) {
            load_pairs<THREADS, BF16>(rd, zd);
            float2 dpart;
            norm_accumulate<true, G::NP>(zt, zd, P.scale_log2, mt, st2, md, sd2, dpart);
            if (rec_draft) {
              const float mw = redux_max(md);
              const float sw =
                  group_sum<5>(__fmul_rn(__fadd_rn(dpart.x, dpart.y), ex2(__fsub_rn(md, mw))));
              if (lane == 0) {
                S2.crec[0][k * NW + warp] = mw;
                S2.crec[1][k * NW + warp] = sw;
              }
            }
            if (zapp) dmin = fminf(dmin, dmin_pairs<G::NP>(zt, zd));
          } else {
            float2 unused;
            const float2 part =
                norm_accumulate<false, G::NP>(zt, zd, P.scale_log2, mt, st2, md, sd2, unused);
            if (rec_ok) {
              // a leaf: its bonus draw samples this row; record the warp's
              // chunk mass against the warp's largest reference
              const float mw = redux_max(mt);
              const float sw =
                  group_sum<5>(__fmul_rn(__fadd_rn(part.x, part.y), ex2(__fsub_rn(mt, mw))));
              if (lane == 0) {
                S2.crec[0][k * NW + warp] = mw;
                S2.crec[1][k * NW + warp] = sw;
              }
            }
          }
          return false;
        });
    if (err) break;
    // A slice of at most S chunks stays in the ring (chunk k in stage k; not
    // in the instance with the optional paths, whose registers it exceeds):
    // every later pass of the visit reads it from shared memory.
    src.held = !VAR && (nloc + G::CE - 1) / G::CE <= (src.rows == 2 ? G::S : 2 * G::S);
    const float st = __fadd_rn(st2.x, st2.y), sd = __fadd_rn(sd2.x, sd2.y);
    if (have_kid) {
      S2.kzt[tid] = kz_t;
      S2.kzd[tid] = kz_d;
    }
    if (mt == kNoRef) mt = -INFINITY;  // no finite logit: the exchange's "no mass" marker
    if (md == kNoRef) md = -INFINITY;
    const bool bad_t = !(st <= FLT_MAX), bad_d = !(sd <= FLT_MAX);
    const int flags = (bad_t ? kFlagTargetBad : 0) | (bad_d ? kFlagDraftBad : 0);
    float o[8];
    int oflags;
    if (zapp) {
#pragma unroll
      for (int off = 16; off; off >>= 1) dmin = fminf(dmin, __shfl_xor_sync(0xffffffffu, dmin, off));
      if ((tid & 31) == 0) H.wpart[tid >> 5][0] = dmin;
      __syncthreads();
      if (tid < 32) {
        float v = tid < NW ? H.wpart[tid][0] : INFINITY;
#pragma unroll
        for (int off = 16; off; off >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, off));
        dmin = v;
      }
      __syncthreads();  // the exchange below reuses H.wpart
    }
    mark(kPhaseNormX);
    exchange<NW, true>(H, mt, st, md, sd, flags, -1, xp, xph, rank, C, o, oflags, dmin);
    mark(kPhaseTest);
    const float dmin_all = H.bc[9];
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
    K.sig = K.invSt;
    if constexpr (SPEC) {
      K.sc = SpecConst{P.scale_log2, P.scale_log2_lo, K.Mt, K.Md, df(0.f)};
      K.tab = S2.tab;
    }
    // SpecInfer: the double-float normalisers (taken at the node's first
    // rejection) and the current residual mass T
    bool spec_norm = false;
    DF spec_Sd = df(0.f), spec_T = df(0.f);
    if (drafting && need_draft) draft_children(c1, K, rbase);
    // Z_applied: Z* = min_{q>0} p / q = 2^(c min(z_t - z_d) - M_t + M_d) S_d / S_t,
    // valid while no map has zeroed a token (after one, Z* = 0)
    const float zstar = zapp ? __fdiv_rn(__fmul_rn(ex2(__fmaf_rn(dmin_all, K.c, __fsub_rn(K.Md, K.Mt))),
                                                   K.invSt),
                                         K.invSd)
                             : 0.f;
    Pending Pm{kScale, -1, 0.f, 0.f, 0.f};  // parameters of the latest map (sampler masses)
    int mass_kind = 1;

    if (!need_draft) {
      // accepted leaf (or a root without children): bonus token from p
      bool to = false;
      if (rec_ok) crec = ChunkRec{1, K.Mt, K.invSt};
      mark(kPhaseDraw);
      if (!stream_sample<THREADS, BF16, SPEC>(H, S2, ring, P, src, K, chain, mass_kind, Pm,
                                              S2.ufin, b, depth, lo, rank, C, xp, xph, to, crec))
        err |= kErrEmpty;
      if (to) err |= kErrTimeout;
      break;
    }
    // ---- sequential accept tests over the children (S3), shaping on reject
    int accepted = -1, acc_tok = -1;
    // scale of the test denominator's unnormalised values D~ (q~ until a
    // proxy replaces it)
    float dsc = K.invSd;
    for (int i = 0, cn = c1; cn >= 0; ++i, cn = next_sib[cn]) {
      if (i == kMaxKids) { err |= kErrFanout; break; }
      const int x = cand_s[cn];
      if (x < 0 || x >= V) { err |= kErrToken; break; }
      const int nm = S2.nmaps;
      const float qt = exp_of(S2.kzd[i], K.c, K.Md);
      float qx = __fmul_rn(qt, K.invSd);
      float Rt = exp_of(S2.kzt[i], K.c, K.Mt);
      if constexpr (SPEC) {
        if (nm > 0) Rt = df_value(spec_residual(S2.kzt[i], S2.kzd[i], K.sc, K.tab));
      } else if (chain == kChainResiDenom) {
        // The exact chain at x: a map that rejected x leaves R(x) = 0 and
        // the denominator's value there unchanged (K(x0) = D(x0)); a later
        // map then gives it R - r = 0.  D~ changes units at every map
        // (mdsc), so keeping its value means rescaling it.
        float D = qt, Rc = Rt, dprev = K.invSd;
        for (int j = 0; j < nm; ++j) {
          const float dj = S2.mdsc[j];
          if (S2.rej[j] == x) {
            Rc = 0.f;
            D = __fdiv_rn(__fmul_rn(D, dprev), dj);
          } else {
            const float2 mp = S2.map[j];
            const float m = fminf(__fmul_rn(mp.x, D), Rc);
            const float t = __fmaf_rn(m, -1.f, Rc);
            Rc = __fmaf_rn(mp.y, t, m);
            D = t;
          }
          dprev = dj;
        }
        Rt = Rc;
        qx = __fmul_rn(D, dprev);
      } else {
        float D = qt;
        Rt = apply_chain<kChainResi>(S2, nm, Rt, D);
        for (int j = 0; j < nm; ++j)
          if (S2.rej[j] == x) Rt = 0.f;
      }
      const float Rx = __fmul_rn(Rt, K.sig);
      const float u = S2.kua[i];
      if (__fmul_rn(u, qx) < Rx) { accepted = cn; acc_tok = x; break; }
      rejects += 1;
      if constexpr (SPEC) {
        // ---- SpecInfer rejection (Eq. 2, Sec. 3): R <- (R - q)_+ / S, kept as
        // the threshold K of r~ = (p~ - K q~)_+ (specinfer.cuh).  The node's
        // first rejection takes S_t and S_d in double-float (one pass);
        // then K_1 = S_t / S_d, later K_{n+1} = K_n + T_n / S_d, and one pass
        // sums T = sum r~ at the new K.
        if (nm >= kMaxMaps) { err |= kErrFanout; break; }
        mark(kPhaseRej);
          const DF Kprev = K.sc.K;
        if (!spec_norm) {
          DF acc[2] = {df(0.f), df(0.f)};
          stream_pass<THREADS, BF16, 2>(ring, src, [&](const unsigned char* rt,
                                                            const unsigned char* rd, int) -> bool {
            unnorm_sum<G::NE>(ChunkRegs<THREADS, BF16>(rt), StageElem<THREADS, BF16>{rt}, K.sc.c_hi,
                              K.sc.c_lo, K.Mt, K.tab, acc[0]);
            unnorm_sum<G::NE>(ChunkRegs<THREADS, BF16>(rd), StageElem<THREADS, BF16>{rd}, K.sc.c_hi,
                              K.sc.c_lo, K.Md, K.tab, acc[1]);
            return false;
          });
          DF tot[2];
          if (!df_exchange<NW, 2>(H, acc, tot, xp, xph, rank, C)) { err |= kErrTimeout; break; }
          spec_norm = true;
          spec_Sd = tot[1];
          K.sc.K = df_div(tot[0], spec_Sd);
        } else {
          K.sc.K = df_add(K.sc.K, df_div(spec_T, spec_Sd));
        }
        DF acc[1] = {df(0.f)};
        // the last child's rejection defines the final distribution: its
        // pass records it (ChunkRec kind 3)
        const bool rec_last = rec_ok && next_sib[cn] < 0;
        stream_pass<THREADS, BF16, 2>(ring, src, [&](const unsigned char* rt,
                                                          const unsigned char* rd, int k) -> bool {
          const float cr = residual_sum<G::NE>(
              ChunkRegs<THREADS, BF16>(rt), ChunkRegs<THREADS, BF16>(rd),
              StageElem<THREADS, BF16>{rt}, StageElem<THREADS, BF16>{rd}, K.sc, K.tab, acc[0]);
          if (rec_last) {
            const float wr = group_sum<5>(cr);
            if (lane == 0) S2.crec[0][k * NW + warp] = wr;
          }
          return false;
        });
        DF tot[1];
        if (!df_exchange<NW, 1>(H, acc, tot, xp, xph, rank, C)) { err |= kErrTimeout; break; }
        mark(kPhaseTest);
        if (tot[0].hi > 0.f) {
          spec_T = tot[0];
          K.sig = __frcp_rn(df_value(spec_T));
          // per-CTA masses of the residual for the draw: the exchange's
          // per-CTA T (head part) times 1 / T
          Pm = Pending{kSpec, x, K.sig, 0.f, 0.f};
          mass_kind = 3;
          if (rec_last) crec = ChunkRec{3, 0.f, K.sig};
          S2.rej[nm] = x;
          S2.nmaps = nm + 1;
        } else {  // degenerate rejection: R is kept unchanged
          K.sc.K = Kprev;
          info |= kInfoDegenerate;
          mass_kind = 0;
        }
        continue;
      }
      // ---- ResiSpec rejection (Algorithm 1, GetProxy)
      float Z = __fsub_rn(qx, Rx);
      if (zapp)  // max(Z*, |gap|), at most 1 - R(x0)
        Z = fminf(fmaxf(nm == 0 ? zstar : 0.f, fabsf(Z)), __fsub_rn(1.f, Rx));
      if (!(Z > 0.f)) {  // degenerate rejection: R is kept unchanged
        info |= kInfoDegenerate;
        continue;
      }
      if (nm >= kMaxMaps) { err |= kErrFanout; break; }
      mark(kPhaseRej);
      // one pass: the residual so far and the sums of the new map, in
      // unnormalised units (k: the new map's scalar).  The rejected tokens
      // get no special case here; their terms are taken out below.
      float kq = __fdiv_rn(__fmul_rn(Z, dsc), K.sig);
      // s1: sum of min(k D~, R~); s2: sum of t, or in a level pass the sum of R~ where
      // D~ > 0 (s1 for an unbounded k); s3 (level pass): the sum of D~ where
      // k D~ < R~, the slope of s1 in k.  All as pairs of lanes.  D~ is q~
      // unless the proxies replace the denominator (then the chain leaves it
      // in q[]).
      float2 s1p, s2p, s3p;
      // the last child's rejection defines the final distribution when it
      // leaves a map: its pass records it (ChunkRec kind 2)
      const bool rec_last = rec_ok && next_sib[cn] < 0;
      auto rej_pass = [&](auto kind_c, auto level_c, auto rec_c) {
        constexpr int KIND = decltype(kind_c)::value;
        constexpr bool LEVEL = decltype(level_c)::value;
        constexpr bool REC = decltype(rec_c)::value;
        const float2 c2 = dup2(K.c), nMt = dup2(-K.Mt), nMd = dup2(-K.Md), kq2 = dup2(kq);
        stream_pass<THREADS, BF16, 2>(ring, src, [&](const unsigned char* rt,
                                                          const unsigned char* rd, int k) -> bool {
          constexpr int NP = G::NP;
          float2 Rv[NP], q[NP];
          load_pairs<THREADS, BF16>(rt, Rv);  // -inf past the slice: 0
          load_pairs<THREADS, BF16>(rd, q);
#pragma unroll
          for (int j = 0; j < NP; ++j) {
            Rv[j] = ex2x2(__ffma2_rn(Rv[j], c2, nMt));
            q[j] = ex2x2(__ffma2_rn(q[j], c2, nMd));
          }
          float2 t[NP];
          apply_chain_pairs<NP, KIND>(S2, nm, Rv, q);
          float2 m[NP];
#pragma unroll
          for (int j = 0; j < NP; ++j) {
            m[j] = min_part2(kq2, q[j], Rv[j]);
            if constexpr (LEVEL) {
              s3p.x += m[j].x < Rv[j].x ? q[j].x : 0.f;
              s3p.y += m[j].y < Rv[j].y ? q[j].y : 0.f;
              t[j] = make_float2(q[j].x > 0.f ? Rv[j].x : 0.f, q[j].y > 0.f ? Rv[j].y : 0.f);
            } else {
              t[j] = __ffma2_rn(m[j], dup2(-1.f), Rv[j]);
            }
          }
          const float2 cm = sum_pairs<NP>(m);
          const float2 ct = sum_pairs<NP>(t);
          s1p = __fadd2_rn(s1p, cm);
          s2p = __fadd2_rn(s2p, ct);
          if constexpr (REC) {
            const float wm = group_sum<5>(__fadd_rn(cm.x, cm.y));
            const float wt = group_sum<5>(__fadd_rn(ct.x, ct.y));
            if (lane == 0) {
              S2.crec[0][k * NW + warp] = wm;
              S2.crec[1][k * NW + warp] = wt;
            }
          }
          return false;
        });
      };
      // The level fill (r = min(lam q, R) with sum r = Z) moves k by Newton
      // steps from k = Z: s1 is concave and piecewise linear in k, so every
      // step stays at or below the level and the steps end on its piece.
      // The loop stops when the deficit is below 2^-22 Z, when a step no
      // longer moves k in fp32, or after kLevelSteps passes; the residual is
      // then normalised by the mass reached, so what is left of the deficit
      // scales every token by the same relative amount (as a rounding
      // would) instead of moving mass between tokens.  When even an
      // unbounded level falls short of Z (the first level pass's s2 < Z: the
      // support of the denominator cannot hold the budget) no level exists:
      // one plain pass at k = FLT_MAX saturates that support and the default
      // fill places the rest on the tokens outside it.  Every CTA sees the
      // same exchanged sums, so all take the same steps.
      constexpr int kLevelSteps = 24;
      const bool level = VAR && P.level_fill != 0;
      bool timed_out = false, saturate = false;
      float s1, s2, s3;
      for (int step = 0;; ++step) {
        const bool lpass = level && !saturate;
        s1p = s2p = s3p = make_float2(0.f, 0.f);
        if (chain == kChainResiDenom) {
          if (lpass)
            rej_pass(std::integral_constant<int, kChainResiDenom>{}, std::true_type{},
                     std::false_type{});
          else
            rej_pass(std::integral_constant<int, kChainResiDenom>{}, std::false_type{},
                     std::false_type{});
        } else if (lpass) {
          rej_pass(std::integral_constant<int, kChainResi>{}, std::true_type{}, std::false_type{});
        } else if (!VAR && rec_last) {
          rej_pass(std::integral_constant<int, kChainResi>{}, std::false_type{}, std::true_type{});
        } else {
          rej_pass(std::integral_constant<int, kChainResi>{}, std::false_type{},
                   std::false_type{});
        }
        s1 = __fadd_rn(s1p.x, s1p.y);
        s2 = __fadd_rn(s2p.x, s2p.y);
        s3 = __fadd_rn(s3p.x, s3p.y);
        {
          // The token just rejected (r(x0) = 0) and the earlier rejected ones
          // (R = 0 there) add nothing: the thread that summed each such token
          // of this slice subtracts the terms the pass gave it, recomputed
          // bit for bit (each distinct token once).
          for (int t = -1; t < nm; ++t) {
            const int y = t < 0 ? x : S2.rej[t];
            const int yk = t < 0 ? i : S2.rejk[t];
            if (y < lo || y >= lo + nloc) continue;
            if ((((y - lo) % G::CE) / VEC) % THREADS != tid) continue;
            bool seen = t >= 0 && y == x;
            for (int t2 = 0; t2 < t && !seen; ++t2) seen = S2.rej[t2] == y;
            if (seen) continue;
            float Dy = exp_of(S2.kzd[yk], K.c, K.Md);
            const float py = exp_of(S2.kzt[yk], K.c, K.Mt);
            const float Ry = chain == kChainResiDenom
                                 ? apply_chain<kChainResiDenom>(S2, nm, py, Dy)
                                 : apply_chain<kChainResi>(S2, nm, py, Dy);
            const float my = fminf(__fmul_rn(kq, Dy), Ry);
            s1 = __fsub_rn(s1, my);
            if (!lpass) {
              s2 = __fsub_rn(s2, __fmaf_rn(my, -1.f, Ry));
            } else {
              if (Dy > 0.f) s2 = __fsub_rn(s2, Ry);
              if (my < Ry) s3 = __fsub_rn(s3, Dy);
            }
          }
        }
        if (lpass)
          exchange<NW, false, 3>(H, s1, s2, s3, 0.f, 0, -1, xp, xph, rank, C, o, oflags);
        else
          exchange<NW, false>(H, s1, s2, 0.f, 0.f, 0, -1, xp, xph, rank, C, o, oflags);
        mark(kPhaseTest);
        if (oflags & kFlagTimeout) { timed_out = true; break; }
        if (!level || saturate || step + 1 >= kLevelSteps) break;
        float kn;
        if (step == 0 && __fmul_rn(o[1], K.sig) < Z) {  // no level reaches Z
          saturate = true;
          kn = FLT_MAX;
        } else {
          // normalised: s1 o[0] sig, slope o[2] sig per unit of k
          const float gap = __fsub_rn(Z, __fmul_rn(o[0], K.sig));
          const float slope = __fmul_rn(o[2], K.sig);
          if (!(gap > __fmul_rn(Z, 0x1p-22f)) || !(slope > 0.f)) break;
          kn = __fadd_rn(kq, __fdiv_rn(gap, slope));
          if (!(kn > kq)) break;
        }
        kq = kn;
        mark(kPhaseRej);
      }
      if (timed_out) { err |= kErrTimeout; break; }
      bool has_map = false;
      float a = 0.f, lam = 0.f;
      {
        const float S1 = __fmul_rn(o[0], K.sig), S2s = __fmul_rn(o[1], K.sig);
        const float delta = __fsub_rn(Z, S1);
        lam = S2s > 0.f && (!level || saturate) ? fminf(fmaxf(__fdiv_rn(delta, S2s), 0.f), 1.f)
                                                 : 0.f;
        const float norm = __fmaf_rn(lam, S2s, S1);
        if (norm > 0.f) {
          has_map = true;
          a = __frcp_rn(norm);
          mass_kind = 2;
        }
      }
      if (has_map && !VAR && rec_last && !level) {
        // The records hold every token's terms; the rejected tokens' residual
        // is 0: thread 0 takes their terms out of their (chunk, warp) records
        // in a fixed order (each distinct token once), recomputed as the pass
        // computed them.
        if (tid == 0)
          for (int t = -1; t < nm; ++t) {
            const int y = t < 0 ? x : S2.rej[t];
            const int yk = t < 0 ? i : S2.rejk[t];
            if (y < lo || y >= lo + nloc) continue;
            bool seen = t >= 0 && y == x;
            for (int t2 = 0; t2 < t && !seen; ++t2) seen = S2.rej[t2] == y;
            if (seen) continue;
            float Dy = exp_of(S2.kzd[yk], K.c, K.Md);
            const float Ry = apply_chain<kChainResi>(S2, nm, exp_of(S2.kzt[yk], K.c, K.Mt), Dy);
            const float my = fminf(__fmul_rn(kq, Dy), Ry);
            const int off = y - lo;
            const int r = (off / G::CE) * NW + ((off % G::CE) / VEC % THREADS) / 32;
            S2.crec[0][r] = __fsub_rn(S2.crec[0][r], my);
            S2.crec[1][r] = __fsub_rn(S2.crec[1][r], __fmaf_rn(my, -1.f, Ry));
          }
        crec = ChunkRec{2, lam, __fmul_rn(K.sig, a)};
      }
      if (has_map) {
        if (chain == kChainResiDenom)  // the proxy (1 - lambda) t~ becomes the denominator
          dsc = __fmul_rn(K.sig, __fsub_rn(1.f, lam));
        K.sig = __fmul_rn(K.sig, a);
        // per-CTA masses of the new residual: (p0 + lambda p1) sig from this
        // exchange's unnormalised partials
        Pm = Pending{kResi, x, K.sig, Z, lam};
        // every thread, identical values (see the visit start)
        S2.map[nm] = make_float2(kq, lam);
        S2.mdsc[nm] = dsc;
        S2.rej[nm] = x;
        S2.rejk[nm] = (int16_t)i;
        S2.nmaps = nm + 1;
      } else {
        info |= kInfoDegenerate;
        mass_kind = 0;  // the exchange's partials do not describe R: sum it directly
      }
    }
    if (err) break;

    if (accepted < 0) {
      // every child rejected: residual draw (Algorithm 1, last step)
      bool to = false;
      mark(kPhaseDraw);
      if (!stream_sample<THREADS, BF16, SPEC>(H, S2, ring, P, src, K, chain, mass_kind, Pm,
                                              S2.ufin, b, depth, lo, rank, C, xp, xph, to, crec))
        err |= kErrEmpty;
      if (to) err |= kErrTimeout;
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
    __syncthreads();  // every read of this visit's S2 state precedes the next visit's writes
  }

  mark(kPhaseSetup);
  if (prof && rank == 0 && tid == 0)
    for (int k = 0; k < kPhases; ++k) P.out_phase[(size_t)b * kPhases + k] = (int64_t)S2.phc[k];
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
