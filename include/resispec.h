/*
 * resispec.h -- C ABI of the ResiSpec verification library (GB300, sm_103a).
 *
 * One call verifies a batch of draft token trees against their target
 * logits, as in the verification step of multi-candidate speculative
 * sampling (paper: "ResiSpec: Enhancing Multi-Candidate Speculative Sampling
 * via Residual Distribution Shaping", Sec. 3 and Algorithm 1):
 *
 *   for every sequence b: start at the root; turn the node's target and
 *   draft logits into tempered distributions p, q (softmax(z / T)); test the
 *   node's children in ascending node order with u < R(x) / q(x), R starting
 *   at p; after each rejection reshape R (ResiSpec: GetProxy of Algorithm 1;
 *   SpecInfer: Eq. 2); on acceptance emit the child's token and descend
 *   into it; when every child is rejected emit x ~ R; when an accepted node
 *   has no children emit a bonus token x ~ p of that node.
 *
 * Conventions for every entry point below:
 *   - Pointers named *_logits, tree_parents, cand_tokens, out_* and status
 *     are DEVICE pointers owned by the caller (e.g. the storage of torch
 *     tensors).  The library allocates no device memory and keeps no
 *     reference to any pointer after the call returns.
 *   - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and the call returns without synchronising.
 *   - Argument errors are returned synchronously as a resispec_status and
 *     nothing is launched.  Errors that depend on device data are reported
 *     on the device (see RESISPEC_ERR_*): the kernel never traps.
 *   - Randomness: u = U(seed, b, row, draw) from Philox4x64-10 (Salmon et
 *     al., SC 2011) with key (seed, 0) and counter (row, b, 0, 0);
 *     u = (word[draw] >> 40) * 2^-24.  The accept test of candidate node c
 *     uses row c+1, draw 0; the residual / bonus draw at the node whose
 *     logits are row r uses row r, draw 1.  Outputs are a pure function of
 *     the inputs, seed and mode.
 */
#ifndef RESISPEC_H_
#define RESISPEC_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define RESISPEC_ABI_VERSION 4

/* Synchronous return codes. */
typedef enum {
  RESISPEC_OK = 0,
  RESISPEC_E_ARG = 1,         /* NULL pointer, temperature not finite or <= 0, bad option */
  RESISPEC_E_SHAPE = 2,       /* a size outside the supported range */
  RESISPEC_E_DTYPE = 3,       /* dtype not RESISPEC_F32 / RESISPEC_BF16 */
  RESISPEC_E_UNSUPPORTED = 4, /* device is not sm_103 or cannot host the cluster */
  RESISPEC_E_CUDA = 5         /* a CUDA runtime call failed; see resispec_last_error() */
} resispec_status;

typedef enum { RESISPEC_F32 = 0, RESISPEC_BF16 = 1 } resispec_dtype;

/* RESISPEC: Algorithm 1 with GetProxy (budget Z = q(x0) - R(x0), deficit
 *   filled in proportion to the remaining capacity R - r off x0).
 * SPECINFER: the residual recurrence R <- (R - q)_+ / sum (Eq. 2, Sec. 3). */
typedef enum { RESISPEC_MODE_RESISPEC = 0, RESISPEC_MODE_SPECINFER = 1 } resispec_mode;

/* Bits of the optional device status word (atomically OR-ed per sequence).
 * A sequence with an ERR bit gets out_accept_len = -1 and an all -1 token
 * row. */
#define RESISPEC_ERR_TREE 1        /* tree_parents[c] not in [-1, c) */
#define RESISPEC_ERR_TOKEN 2       /* a tested candidate token outside [0, V) */
#define RESISPEC_ERR_NONFINITE 4   /* NaN or +inf in a visited logit row */
#define RESISPEC_ERR_EMPTY_ROW 8   /* a visited row (or the residual) has no mass */
#define RESISPEC_ERR_DEPTH 16      /* more accepted tokens than max_depth */
#define RESISPEC_ERR_TIMEOUT 32    /* a bounded wait for a row copy gave up */
#define RESISPEC_ERR_FANOUT 64     /* streaming kernel: the walk reached child
                                      RESISPEC_MAX_FANOUT_STREAM + 1 of a node (it
                                      tests at most that many children per node) */
#define RESISPEC_INFO_DEGENERATE 256 /* informational: a rejection left R unchanged */

/* Phases of out_phase_cycles.  The paper splits ResiSpec's cost into
 * budgeting, redistribution and proxy formulation: budgeting is part of
 * RESISPEC_PHASE_TEST, redistribution is RESISPEC_PHASE_REJECT, and the
 * proxy is never materialised (R' = r / Z directly). */
#define RESISPEC_PHASE_SETUP 0     /* before the first pass (setup overlaps it) */
#define RESISPEC_PHASE_NORM 1      /* normaliser passes */
#define RESISPEC_PHASE_NORM_X 2    /* their cluster exchanges */
#define RESISPEC_PHASE_TEST 3      /* accept tests and budgets */
#define RESISPEC_PHASE_REJECT 4    /* rejection passes and their exchanges */
#define RESISPEC_PHASE_DRAW 5      /* residual / bonus draw */
#define RESISPEC_PHASES 6

#define RESISPEC_MAX_VOCAB 262144
#define RESISPEC_MAX_NODES 4096
#define RESISPEC_MAX_FANOUT_STREAM 128

/* Sizes of one call.  Logit rows: row 0 is the root, row j+1 is node j. */
typedef struct {
  int32_t batch;     /* B >= 0 sequences (B = 0 launches nothing) */
  int32_t num_nodes; /* N in [0, RESISPEC_MAX_NODES] tree nodes, root excluded */
  int32_t vocab;     /* V in [1, RESISPEC_MAX_VOCAB] */
  int32_t max_depth; /* D >= 0; out_tokens has D + 1 columns */
  int32_t dtype;     /* resispec_dtype of both logit arrays */
} resispec_dims;

#define RESISPEC_FLAG_NO_TMA 1   /* force plain loads instead of bulk copies */
#define RESISPEC_FLAG_PREFETCH 2 /* resident kernel: warm L2 with the first child's rows */
#define RESISPEC_FLAG_RESIDENT 4 /* force the resident kernel */
#define RESISPEC_FLAG_STREAM 8   /* force the streaming kernel */
#define RESISPEC_FLAG_Z_APPLIED 16 /* RESISPEC mode budget variant (Sec. 5.3 heuristic):
                                      Z = max(Z*, |q(x0) - R(x0)|), Z* = min over
                                      q > 0 of R/q (0 once a map of the node has
                                      zeroed a token), clamped to Z <= 1 - R(x0);
                                      streaming kernel only (combined with
                                      RESISPEC_FLAG_RESIDENT: RESISPEC_E_ARG) */
#define RESISPEC_FLAG_PROXY_DENOM 32 /* RESISPEC mode variant (the paper's EAGLE
                                      integration, App. C): after each rejection
                                      the test denominator becomes that rejection's
                                      proxy K (K = R - r off x0, K(x0) = D(x0)),
                                      and the next GetProxy takes it in place of
                                      q; candidates stay draws from q.  Streaming
                                      kernel only (with RESISPEC_FLAG_RESIDENT:
                                      RESISPEC_E_ARG); no effect in SPECINFER mode */
#define RESISPEC_FLAG_LEVEL_FILL 64 /* RESISPEC mode variant of GetProxy's step 3
                                      (Algorithm 1; the paper fixes only that the
                                      deficit goes to tokens below their capacity):
                                      r = min(lam q, R) off x0 with the level lam
                                      at which sum r = Z, instead of the default
                                      fill in proportion to the capacity R - r.
                                      lam is found by Newton steps from lam = Z on
                                      the concave, piecewise linear sum (one more
                                      pass over the rows per step, typically 2 to
                                      6 steps); the residual is normalised by the
                                      mass reached (a deficit left below 2^-22 Z
                                      acts as a relative rounding).  When the
                                      support of q cannot hold Z (no level
                                      exists) that support is saturated and the
                                      default rule places the rest.  Streaming
                                      kernel only (with RESISPEC_FLAG_RESIDENT:
                                      RESISPEC_E_ARG); no effect in SPECINFER mode */

/* Kernels.  Both compute the same verification; they differ in where a
 * visited node's rows live between the passes of a visit.
 *   RESIDENT: both rows of the sequence's vocabulary slice stay in the
 *     shared memory of the cluster's CTAs as fp32 (8 bytes per vocabulary
 *     entry per sequence), so only as many sequences as fit on chip run at
 *     once.  Any fan-out.  RESISPEC mode only (SPECINFER with
 *     RESISPEC_FLAG_RESIDENT: RESISPEC_E_ARG).
 *   STREAM: nothing but per-sequence scalars stays on chip; every pass
 *     streams the rows from global memory (the passes after a visit's first
 *     read them from L2, or from shared memory when a CTA's slice fits its
 *     copy ring).  All sequences of a large batch run at once.  Fan-out up
 *     to RESISPEC_MAX_FANOUT_STREAM children per node.
 * The automatic choice is STREAM (measured as fast or faster at every batch
 * size); RESIDENT runs when RESISPEC_FLAG_RESIDENT asks for it. */
#define RESISPEC_KERNEL_RESIDENT 0
#define RESISPEC_KERNEL_STREAM 1

typedef struct {
  int32_t mode;          /* resispec_mode */
  int32_t cluster_size;  /* CTAs per sequence (one thread-block cluster): 0 = automatic
                            (most SMs engaged for this batch), else 1 .. 16 */
  int32_t block_threads; /* 0 = automatic, else 256 or 512 */
  int32_t flags;         /* RESISPEC_FLAG_* */
  int64_t seq_stride;    /* elements between sequences in both logit arrays;
                            -1 = (N + 1) * V; 0 shares one set of rows */
  int32_t* status;       /* optional device int32 OR-ed with RESISPEC_ERR_* bits */
  int32_t* out_nodes;    /* optional device [B, D] accepted node ids, -1 padded */
  float* out_dist;       /* optional device [B, V] fp32: the distribution the
                            last emitted token was drawn from (final residual
                            R, or p of the accepted leaf) */
  int32_t* out_rejects;  /* optional device [B] number of rejections */
  int64_t* out_phase_cycles; /* optional device [B, RESISPEC_PHASES] int64: SM
                                cycles (clock64 on the sequence's first CTA)
                                spent per phase, RESISPEC_PHASE_*; asking for
                                it selects the streaming kernel */
  int32_t* out_candidates; /* optional device [B, N] int32: drafting mode.  The
                              children of every visited node are drawn from that
                              node's tempered draft distribution (Algorithm 1,
                              "x_1..x_k ~ Q i.i.d.": inverse CDF over ascending
                              token ids, child c with u = word 2 of the Philox
                              block of row c + 1) and written here (-1 for the
                              nodes whose parent is not visited); cand_tokens is
                              then not read (may be NULL).  Selects the
                              streaming kernel */
  int64_t parents_stride; /* int32 elements between sequences' trees in
                             tree_parents: 0 (default) = one tree [N] shared by
                             every sequence; N = tree_parents is [B, N], a tree
                             per sequence (dynamic trees; a bad tree marks only
                             its own sequence with RESISPEC_ERR_TREE) */
} resispec_opts;

/* Fills *opts with the defaults (RESISPEC mode, automatic launch shape,
 * seq_stride -1, no optional outputs). */
void resispec_opts_default(resispec_opts* opts);

/* Verify a batch of draft trees (Sec. 3; Algorithm 1; GetProxy).
 *   target_logits  [B, N+1, V] dtype, row-major, 16-byte aligned for the
 *                  bulk-copy path (otherwise plain loads are used)
 *   draft_logits   [B, N+1, V] same layout
 *   tree_parents   [N] int32, parent of node c (-1 = root), parent < c;
 *                  siblings are tested in ascending node index (with
 *                  opts->parents_stride = N: [B, N], one tree per sequence)
 *   cand_tokens    [B, N] int32, token proposed at node c (drawn i.i.d. from
 *                  the parent's tempered draft distribution by the caller)
 *   temperature    T > 0, applied to target and draft logits alike
 *   seed           Philox key (see the header comment)
 *   out_tokens     [B, D+1] int32: accepted tokens, then the residual / bonus
 *                  token, then -1 padding
 *   out_accept_len [B] int32: number of accepted candidates (-1 on a
 *                  per-sequence data error)
 * Uses RESISPEC mode, automatic launch shape and one shared tree. */
int resispec_verify(const void* target_logits, const void* draft_logits,
                    const int32_t* tree_parents, const int32_t* cand_tokens,
                    float temperature, uint64_t seed, int32_t* out_tokens,
                    int32_t* out_accept_len, resispec_dims dims, void* stream);

/* resispec_verify with options (mode, launch shape, stride, optional
 * outputs).  opts may be NULL (defaults). */
int resispec_verify_ex(const void* target_logits, const void* draft_logits,
                       const int32_t* tree_parents, const int32_t* cand_tokens,
                       float temperature, uint64_t seed, int32_t* out_tokens,
                       int32_t* out_accept_len, resispec_dims dims,
                       const resispec_opts* opts, void* stream);

/* Launch shape chosen for a call. */
typedef struct {
  int32_t kernel;          /* RESISPEC_KERNEL_* */
  int32_t cluster_size;    /* CTAs per sequence */
  int32_t block_threads;   /* threads per CTA */
  int32_t smem_bytes;      /* dynamic shared memory per CTA */
  int32_t slice_elems;     /* vocabulary entries per CTA */
  int32_t uses_tma;        /* 1 if rows are fetched with bulk (TMA) copies: the
                              resident kernel on 16-byte aligned rows */
  int32_t vector_loads;    /* 1 if rows move in 16-byte vectors (bulk copies in
                              the resident kernel, per-thread asynchronous
                              16-byte copies in the streaming kernel), 0 if
                              element by element (rows not 16-byte aligned) */
  int32_t active_clusters; /* clusters of this shape resident at once on the
                              current device (0 without a device) */
} resispec_plan_info;

/* Launch shape resispec_verify_ex would use for these sizes and options on
 * the current device (no launch; without a usable device a size-only rule
 * is applied).  Returns the same argument errors as resispec_verify_ex. */
int resispec_plan(resispec_dims dims, const resispec_opts* opts, resispec_plan_info* out);

/* Device Philox draws for testing the counter-based generator: for i < n,
 * u0[i] = U(seed, seq[i], row[i], 0) and u1[i] = U(seed, seq[i], row[i], 1).
 * seq, row, u0, u1 are device arrays of length n. */
int resispec_uniforms(uint64_t seed, const int32_t* seq, const int32_t* row,
                      int32_t n, float* u0, float* u1, void* stream);

/* Text of a status code / of the last CUDA error seen by this thread. */
const char* resispec_status_string(int status);
const char* resispec_last_error(void);

int resispec_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* RESISPEC_H_ */
