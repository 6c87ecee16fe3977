// Host side of the C ABI declared in include/resispec.h: argument checks,
// launch planning (kernel, cluster size, threads, shared memory) and the
// cluster launch of the fused verification kernel on the caller's stream.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <map>
#include <mutex>
#include <tuple>

#include "../../include/resispec.h"
#include "kernels.h"
#include "verify_stream.cuh"

namespace rs {

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

namespace {

thread_local char g_last_error[256] = "";

void set_error(const char* what, cudaError_t e) {
  snprintf(g_last_error, sizeof g_last_error, "%s: %s (%d)", what, cudaGetErrorString(e),
           (int)e);
}

constexpr int kMaxSmem = 227 * 1024;      // dynamic shared memory per CTA on sm_10x
constexpr int kAutoSliceBytes = 96 * 1024; // target on-chip bytes per CTA (two fp32 rows)

struct Plan {
  int kernel = RESISPEC_KERNEL_RESIDENT;
  int var = 0;  // streaming kernel with the optional paths compiled in
  int spec = 0; // streaming kernel, SpecInfer instance
  int C = 1;
  int threads = 512;
  int L = 8;
  int npad = 16;
  int smem = 0;
  int use_tma = 0;
  int active = 0;
};

int round_up(int x, int m) { return (x + m - 1) / m * m; }

int slice_for(int V, int C) { return round_up((V + C - 1) / C, 8); }

// Head, two fp32 rows, then the tree: parent / first child / next sibling
// (int16), the candidate tokens of the sequence (int32) and two uniforms per
// logit row (fp32).
int tree_bytes(int npad) { return npad * 2 + (npad + 16) * 2 + npad * 2 + npad * 4 + npad * 8; }

int smem_for(int L, int npad) { return round_up(rs::kHeadBytes + 8 * L + tree_bytes(npad), 128); }

// Streaming kernel: head, stream head, the cp.async ring (96 KB at 512
// threads; the sampler's chunk buffer reuses one of its stages), then the
// tree (parents, first children, next siblings, candidate tokens; the
// uniforms are drawn per visit).
int stream_smem_for(int threads, bool bf16, int npad) {
  const int ring = bf16 ? rs::StreamGeom<512, true>::RING : rs::StreamGeom<512, false>::RING;
  const int tree = npad * 2 + (npad + 16) * 2 + npad * 2 + npad * 4;
  return round_up(rs::kHeadBytes + rs::kStreamHeadBytes + ring * threads / 512 + tree, 128);
}

struct DeviceInfo {
  int sms = 0;
  int major = 0;
  int minor = 0;
};

std::mutex g_mu;
DeviceInfo g_dev[64];
bool g_attr_set[64][32];

int query_device(int* dev_out, DeviceInfo* info) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) { set_error("cudaGetDevice", e); return RESISPEC_E_CUDA; }
  if (dev < 0 || dev >= 64) return RESISPEC_E_UNSUPPORTED;
  std::lock_guard<std::mutex> lk(g_mu);
  DeviceInfo& d = g_dev[dev];
  if (d.sms == 0) {
    cudaDeviceProp prop;
    e = cudaGetDeviceProperties(&prop, dev);
    if (e != cudaSuccess) { set_error("cudaGetDeviceProperties", e); return RESISPEC_E_CUDA; }
    d.sms = prop.multiProcessorCount;
    d.major = prop.major;
    d.minor = prop.minor;
  }
  *dev_out = dev;
  *info = d;
  return RESISPEC_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int check_dims(const resispec_dims& d) {
  if (d.batch < 0 || d.num_nodes < 0 || d.max_depth < 0) return RESISPEC_E_SHAPE;
  if (d.vocab < 1 || d.vocab > RESISPEC_MAX_VOCAB) return RESISPEC_E_SHAPE;
  if (d.num_nodes > RESISPEC_MAX_NODES) return RESISPEC_E_SHAPE;
  if (d.max_depth > d.num_nodes) return RESISPEC_E_SHAPE;
  if (d.dtype != RESISPEC_F32 && d.dtype != RESISPEC_BF16) return RESISPEC_E_DTYPE;
  return RESISPEC_OK;
}

// Clusters of this shape that can be resident at once (0: the shape cannot
// be launched).  Cached per device and shape.
using OccKey = std::tuple<int, int, int, int, int, int>;  // dev, kernel id, threads, bf16, C, smem
std::map<OccKey, int> g_occ;

template <int THREADS, bool BF16>
const void* kernel_ptr(int kernel, int var, int spec) {
  if (kernel == RESISPEC_KERNEL_STREAM && var)
    return BF16 ? rs::stream_var_entry_bf16(THREADS, spec) : rs::stream_var_entry_f32(THREADS, spec);
  if (kernel == RESISPEC_KERNEL_STREAM)
    return BF16 ? rs::stream_entry_bf16(THREADS, spec) : rs::stream_entry_f32(THREADS, spec);
  return BF16 ? rs::resident_entry_bf16(THREADS) : rs::resident_entry_f32(THREADS);
}

template <int THREADS, bool BF16>
int query_clusters(int kernel, int var, int spec, int C, int smem) {
  const void* kern = kernel_ptr<THREADS, BF16>(kernel, var, spec);
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem) !=
          cudaSuccess ||
      cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
          cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = dim3((unsigned)(C * 64), 1, 1);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = (size_t)smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, (void*)kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

int active_clusters(int dev, int kernel, int var, int spec, int threads, bool bf16, int C,
                    int smem) {
  const OccKey key{dev, kernel * 4 + (var ? 1 : 0) + (spec ? 2 : 0), threads, bf16 ? 1 : 0, C,
                   smem};
  {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_occ.find(key);
    if (it != g_occ.end()) return it->second;
  }
  int n;
  if (threads == 512)
    n = bf16 ? query_clusters<512, true>(kernel, var, spec, C, smem)
             : query_clusters<512, false>(kernel, var, spec, C, smem);
  else
    n = bf16 ? query_clusters<256, true>(kernel, var, spec, C, smem)
             : query_clusters<256, false>(kernel, var, spec, C, smem);
  std::lock_guard<std::mutex> lk(g_mu);
  g_occ[key] = n;
  return n;
}

// Resident kernel: cluster size.  With a device, most SMs engaged (resident
// clusters capped by the batch, times their size; ties go to the larger
// cluster, which shortens a sequence's latency).
int plan_resident(const resispec_dims& d, int cs, int dev, int sms, Plan* p) {
  const int V = d.vocab;
  const bool bf16 = d.dtype == RESISPEC_BF16;
  if (cs) {
    p->C = cs;
  } else if (dev >= 0) {
    int best = 0;
    int64_t best_score = -1;
    for (int C = 1; C <= rs::kMaxCluster; ++C) {
      const int smem = smem_for(slice_for(V, C), p->npad);
      if (smem > kMaxSmem) continue;
      const int n =
          active_clusters(dev, RESISPEC_KERNEL_RESIDENT, 0, 0, p->threads, bf16, C, smem);
      if (n <= 0) continue;
      const int64_t score = std::min<int64_t>(d.batch, n) * C;
      if (score >= best_score) { best_score = score; best = C; }
    }
    if (best == 0) return RESISPEC_E_UNSUPPORTED;
    p->C = best;
  } else {
    int C = 1;
    while (C < 16 && 8 * slice_for(V, C) > kAutoSliceBytes) C *= 2;
    while (sms > 0 && C < 16 && (int64_t)d.batch * C * 2 <= sms) C *= 2;
    p->C = C;
  }
  p->L = slice_for(V, p->C);
  p->smem = smem_for(p->L, p->npad);
  if (p->smem > kMaxSmem) return RESISPEC_E_SHAPE;
  p->active = dev >= 0 ? active_clusters(dev, RESISPEC_KERNEL_RESIDENT, 0, 0, p->threads, bf16,
                                         p->C, p->smem)
                       : 0;
  return RESISPEC_OK;
}

// Streaming kernel: block size and cluster size.  A sequence's passes
// shrink as 1 / C, and the batch runs in ceil(B / n) waves of n resident
// clusters (per-sequence chains differ in length, so the longest chain, run
// at C CTAs, sets the time).  Measured on GB300 (eleven workloads, both
// block sizes):
//  - 256-thread CTAs (three per SM, half the ring each) beat 512-thread ones
//    on trees with about two children per node (N^(1/D) <= 2.5: binary
//    depth-5 trees 102.7 against 107.9 us at B = 64, single position k = 2
//    at B = 128 85.8 against 104.4 us) and on shallow trees of at most 4
//    nodes (single position k = 4 at B = 128: 92.7 against 107.5 us), where
//    a sequence spends its time in normaliser passes rather than in
//    rejection passes; wider trees and batches that fit 16-CTA clusters of
//    512 threads keep 512.
//  - Trees deeper than 2 levels take the largest C that runs the batch in
//    one wave; when that leaves more than 128 elements per thread and row in
//    a CTA's slice, the largest C within two waves (tree488 at B = 128:
//    clusters of 4 in two waves 256.6 us, of 2 in one wave 288.8 us).
//  - Shallow trees at 512 threads (up to 2 levels: few visits, many
//    rejection passes) accept up to 4 waves, clusters of 16 up to 2.
// Without a device, 2 CTAs of 512 threads or 3 of 256 per SM on 152 SMs
// are assumed and a cluster of 16 is taken to fit 14 times per 304 CTA
// slots (how many clusters of 16 CTAs GB300 places at once), smaller ones in
// proportion.
int plan_stream(const resispec_dims& d, int cs, bool auto_threads, int dev, int sms, Plan* p) {
  const bool bf16 = d.dtype == RESISPEC_BF16;
  const int B = std::max(d.batch, 1);
  auto active_for = [&](int T, int C) {
    const int smem = stream_smem_for(T, bf16, p->npad);
    if (dev >= 0)
      return active_clusters(dev, RESISPEC_KERNEL_STREAM, p->var, p->spec, T, bf16, C, smem);
    const int slots = (sms > 0 ? sms : 152) * (T >= 512 ? 2 : 3);
    return C == 16 ? 14 * slots / 304 : slots / C;
  };
  if (auto_threads) {
    const double g = d.max_depth > 0
                         ? std::pow((double)std::max(d.num_nodes, 1), 1.0 / d.max_depth)
                         : 1e30;
    const bool narrow = g <= 2.5 || (d.max_depth <= 2 && d.num_nodes <= 4);
    p->threads = (narrow && B > active_for(512, 16)) ? 256 : 512;
  }
  const int T = p->threads;
  p->smem = stream_smem_for(T, bf16, p->npad);
  if (p->smem > kMaxSmem) return RESISPEC_E_SHAPE;
  if (cs) {
    p->C = cs;
  } else {
    auto waves = [&](int C) {
      const int n = active_for(T, C);
      return n > 0 ? (B + n - 1) / n : INT_MAX;
    };
    int best = 0;
    if (T == 512 && d.max_depth <= 2) {
      for (int C : {16, 8, 4, 2, 1}) {
        if (waves(C) <= (C == 16 ? 2 : 4) || C == 1) {
          best = C;
          break;
        }
      }
    } else {
      static const int kCands[] = {16, 12, 8, 6, 4, 3, 2, 1};
      for (int C : kCands)
        if (waves(C) <= 1 || C == 1) {
          best = C;
          break;
        }
      if (slice_for(d.vocab, best) > 128 * T)
        for (int C : kCands)
          if (C > best && waves(C) <= 2) {
            best = C;
            break;
          }
    }
    p->C = best;
  }
  p->L = slice_for(d.vocab, p->C);
  p->active = dev >= 0 ? active_for(T, p->C) : 0;
  return RESISPEC_OK;
}

// Launch shape.  dev < 0 means no device to query: the automatic choices
// then follow size-only rules.
int make_plan(const resispec_dims& d, const resispec_opts& o, int dev, int sms,
              const void* zt, const void* zd, Plan* p) {
  int st = check_dims(d);
  if (st) return st;
  if (o.mode != RESISPEC_MODE_RESISPEC && o.mode != RESISPEC_MODE_SPECINFER) return RESISPEC_E_ARG;
  if (o.block_threads != 0 && o.block_threads != 256 && o.block_threads != 512)
    return RESISPEC_E_ARG;
  const int cs = o.cluster_size;
  if (cs < 0 || cs > rs::kMaxCluster) return RESISPEC_E_ARG;
  if (o.seq_stride < -1) return RESISPEC_E_ARG;
  if (o.parents_stride < 0) return RESISPEC_E_ARG;
  const bool force_res = (o.flags & RESISPEC_FLAG_RESIDENT) != 0;
  const bool variant = (o.flags & (RESISPEC_FLAG_Z_APPLIED | RESISPEC_FLAG_PROXY_DENOM |
                                   RESISPEC_FLAG_LEVEL_FILL)) != 0 ||
                       o.out_phase_cycles != nullptr || o.out_candidates != nullptr;
  // SpecInfer runs on the streaming kernel only: its residual is evaluated
  // from the raw logits (specinfer.cuh), which the resident kernel does not
  // keep
  const bool spec = o.mode == RESISPEC_MODE_SPECINFER;
  const bool force_str = (o.flags & RESISPEC_FLAG_STREAM) != 0 || variant || spec;
  if (force_res && force_str) return RESISPEC_E_ARG;
  p->var = variant ? 1 : 0;
  p->spec = spec ? 1 : 0;
  p->threads = o.block_threads ? o.block_threads : 512;
  p->npad = round_up(d.num_nodes + 1, 16);
  // The automatic choice is the streaming kernel: measured on GB300 it is
  // as fast or faster at every batch size, also where the whole batch would
  // fit the resident kernel's shared memory (one sequence of 60 nodes at
  // V = 32000: 33 us against 36 us; 16 chains at V = 128256: 49 us against
  // 58 us).  The resident kernel runs when it is asked for.
  if (force_res) {
    p->kernel = RESISPEC_KERNEL_RESIDENT;
    st = plan_resident(d, cs, dev, sms, p);
  } else {
    p->kernel = RESISPEC_KERNEL_STREAM;
    st = plan_stream(d, cs, o.block_threads == 0, dev, sms, p);
  }
  if (st) return st;
  const int64_t es = d.dtype == RESISPEC_BF16 ? 2 : 4;
  const int64_t V = d.vocab;
  const int64_t stride = o.seq_stride < 0 ? (int64_t)(d.num_nodes + 1) * V : o.seq_stride;
  p->use_tma = !(o.flags & RESISPEC_FLAG_NO_TMA) && (V * es) % 16 == 0 &&
               (stride * es) % 16 == 0 && (zt == nullptr || aligned16(zt)) &&
               (zd == nullptr || aligned16(zd));
  return RESISPEC_OK;
}

template <int THREADS, bool BF16>
cudaError_t launch_verify(const Plan& pl, const rs::VerifyParams& prm, cudaStream_t stream,
                          int dev) {
  const void* kern = kernel_ptr<THREADS, BF16>(pl.kernel, pl.var, pl.spec);
  const int slot = (pl.spec ? 16 : 0) + (pl.var ? 8 : 0) +
                   (pl.kernel == RESISPEC_KERNEL_STREAM ? 4 : 0) + (THREADS == 512 ? 2 : 0) +
                   (BF16 ? 1 : 0);
  {
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_attr_set[dev][slot]) {
      cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
      if (e != cudaSuccess) return e;
      e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
      if (e != cudaSuccess) return e;
      g_attr_set[dev][slot] = true;
    }
  }
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.gridDim = dim3((unsigned)(prm.B * pl.C), 1, 1);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = (size_t)pl.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)pl.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // Programmatic dependent launch: the kernel may be scheduled while the
  // preceding kernel on the stream drains; it reads nothing before that
  // kernel has completed (griddepcontrol.wait at its entry), so the
  // stream's ordering is unchanged.
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  void* args[] = {const_cast<rs::VerifyParams*>(&prm)};
  return cudaLaunchKernelExC(&cfg, kern, args);
}

}  // namespace

extern "C" {

void resispec_opts_default(resispec_opts* o) {
  if (!o) return;
  memset(o, 0, sizeof *o);
  o->mode = RESISPEC_MODE_RESISPEC;
  o->seq_stride = -1;
}

int resispec_abi_version(void) { return RESISPEC_ABI_VERSION; }

const char* resispec_status_string(int s) {
  switch (s) {
    case RESISPEC_OK: return "ok";
    case RESISPEC_E_ARG: return "invalid argument";
    case RESISPEC_E_SHAPE: return "size outside the supported range";
    case RESISPEC_E_DTYPE: return "unsupported dtype";
    case RESISPEC_E_UNSUPPORTED: return "unsupported device";
    case RESISPEC_E_CUDA: return "CUDA runtime error";
    default: return "unknown status";
  }
}

const char* resispec_last_error(void) { return g_last_error; }

int resispec_plan(resispec_dims dims, const resispec_opts* opts, resispec_plan_info* out) {
  resispec_opts o;
  resispec_opts_default(&o);
  if (opts) o = *opts;
  int sms = 0;
  int dev = -1;
  DeviceInfo info;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) == cudaSuccess && ndev > 0 && query_device(&dev, &info) == 0 &&
      info.major == 10 && info.minor == 3) {
    sms = info.sms;
  } else {
    dev = -1;
    cudaGetLastError();  // clear a sticky "no device" error
  }
  Plan p;
  const int st = make_plan(dims, o, dev, sms, nullptr, nullptr, &p);
  if (st) return st;
  if (out) {
    out->kernel = p.kernel;
    out->cluster_size = p.C;
    out->block_threads = p.threads;
    out->smem_bytes = p.smem;
    out->slice_elems = p.L;
    out->uses_tma = p.kernel == RESISPEC_KERNEL_RESIDENT ? p.use_tma : 0;
    out->vector_loads = p.use_tma;
    out->active_clusters = p.active;
  }
  return RESISPEC_OK;
}

int resispec_verify_ex(const void* target_logits, const void* draft_logits,
                       const int32_t* tree_parents, const int32_t* cand_tokens,
                       float temperature, uint64_t seed, int32_t* out_tokens,
                       int32_t* out_accept_len, resispec_dims dims,
                       const resispec_opts* opts, void* stream) {
  resispec_opts o;
  resispec_opts_default(&o);
  if (opts) o = *opts;
  int st = check_dims(dims);
  if (st) return st;
  if (!(temperature > 0.f) || !isfinite(temperature)) return RESISPEC_E_ARG;
  if (dims.batch == 0) return RESISPEC_OK;
  if (!target_logits || !draft_logits || !out_tokens || !out_accept_len) return RESISPEC_E_ARG;
  if (dims.num_nodes > 0 && (!tree_parents || (!cand_tokens && !o.out_candidates)))
    return RESISPEC_E_ARG;
  int dev = 0;
  DeviceInfo info;
  st = query_device(&dev, &info);
  if (st) return st;
  if (info.major != 10 || info.minor != 3) {
    snprintf(g_last_error, sizeof g_last_error, "device is sm_%d%d, library is built for sm_103a",
             info.major, info.minor);
    return RESISPEC_E_UNSUPPORTED;
  }
  Plan pl;
  st = make_plan(dims, o, dev, info.sms, target_logits, draft_logits, &pl);
  if (st) return st;
  if ((int64_t)dims.batch * pl.C > 0x7fffffffLL) return RESISPEC_E_SHAPE;

  rs::VerifyParams prm;
  memset(&prm, 0, sizeof prm);
  prm.zt = target_logits;
  prm.zd = draft_logits;
  prm.parents = tree_parents;
  prm.cand = cand_tokens;
  prm.out_tokens = out_tokens;
  prm.out_len = out_accept_len;
  prm.out_nodes = o.out_nodes;
  prm.out_dist = o.out_dist;
  prm.out_rejects = o.out_rejects;
  prm.out_phase = o.out_phase_cycles;
  prm.draft_out = o.out_candidates;
  prm.status = o.status;
  prm.seq_stride = o.seq_stride < 0 ? (int64_t)(dims.num_nodes + 1) * dims.vocab : o.seq_stride;
  prm.parents_stride = o.parents_stride;
  prm.seed = seed;
  {
    // log2(e) / T as an fp32 head and the fp32 rounding of the rest, and the
    // table 2^(j/64) as head + rest (the SpecInfer instance's double-float
    // exponentials)
    const double c = 1.4426950408889634 / (double)temperature;
    prm.scale_log2 = (float)c;
    prm.scale_log2_lo = (float)(c - (double)prm.scale_log2);
    for (int j = 0; j < rs::kExp2Tab; ++j) {
      const double t = exp2((double)(j - 32) / 64.0);
      prm.exp2_tab[j][0] = (float)t;
      prm.exp2_tab[j][1] = (float)(t - (double)prm.exp2_tab[j][0]);
    }
  }
  prm.B = dims.batch;
  prm.N = dims.num_nodes;
  prm.V = dims.vocab;
  prm.D = dims.max_depth;
  prm.slice = pl.L;
  prm.npad = pl.npad;
  prm.mode = o.mode;
  prm.use_tma = pl.use_tma;
  prm.prefetch = (o.flags & RESISPEC_FLAG_PREFETCH) != 0;
  prm.z_applied = (o.flags & RESISPEC_FLAG_Z_APPLIED) != 0;
  prm.denom_update = (o.flags & RESISPEC_FLAG_PROXY_DENOM) != 0;
  prm.level_fill = (o.flags & RESISPEC_FLAG_LEVEL_FILL) != 0;

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  const bool bf16 = dims.dtype == RESISPEC_BF16;
  if (pl.threads == 512)
    e = bf16 ? launch_verify<512, true>(pl, prm, s, dev) : launch_verify<512, false>(pl, prm, s, dev);
  else
    e = bf16 ? launch_verify<256, true>(pl, prm, s, dev) : launch_verify<256, false>(pl, prm, s, dev);
  if (e != cudaSuccess) {
    set_error("verify launch", e);
    return RESISPEC_E_CUDA;
  }
  return RESISPEC_OK;
}

int resispec_verify(const void* target_logits, const void* draft_logits,
                    const int32_t* tree_parents, const int32_t* cand_tokens, float temperature,
                    uint64_t seed, int32_t* out_tokens, int32_t* out_accept_len,
                    resispec_dims dims, void* stream) {
  return resispec_verify_ex(target_logits, draft_logits, tree_parents, cand_tokens, temperature,
                            seed, out_tokens, out_accept_len, dims, nullptr, stream);
}

int resispec_uniforms(uint64_t seed, const int32_t* seq, const int32_t* row, int32_t n,
                      float* u0, float* u1, void* stream) {
  if (n < 0) return RESISPEC_E_SHAPE;
  if (n == 0) return RESISPEC_OK;
  if (!seq || !row || !u0 || !u1) return RESISPEC_E_ARG;
  const int threads = 256;
  rs::uniforms_kernel<<<(n + threads - 1) / threads, threads, 0,
                        static_cast<cudaStream_t>(stream)>>>(seed, seq, row, n, u0, u1);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_error("uniforms launch", e);
    return RESISPEC_E_CUDA;
  }
  return RESISPEC_OK;
}

}  // extern "C"
