"""The C ABI without a GPU: the library builds and loads, exports every
function include/resispec.h declares, and rejects bad arguments
synchronously (before any device work)."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2608_24411_gb300 as rs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "resispec.h")


@pytest.fixture(scope="module")
def lib():
    rs.build()
    return rs.load_library()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\s*\*?\s*(resispec_[a-z_0-9]+)\s*\(", text,
                       flags=re.M)
    return sorted(set(names))


def test_header_declares_entry_points():
    names = declared_functions()
    for n in ("resispec_verify", "resispec_verify_ex", "resispec_plan", "resispec_uniforms",
              "resispec_opts_default", "resispec_status_string", "resispec_last_error",
              "resispec_abi_version"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for n in declared_functions():
        assert hasattr(lib, n), n
    assert set(rs.EXPORTED) <= set(declared_functions())
    assert lib.resispec_abi_version() == 4


def test_opts_default_layout(lib):
    o = rs.Opts()
    ctypes.memset(ctypes.byref(o), 0x5A, ctypes.sizeof(o))
    lib.resispec_opts_default(ctypes.byref(o))
    assert o.mode == 0 and o.cluster_size == 0 and o.block_threads == 0 and o.flags == 0
    assert o.seq_stride == -1
    assert not o.status and not o.out_nodes and not o.out_dist and not o.out_rejects


def _call(lib, dims, T=1.0, null=False, opts=None):
    p = None if null else ctypes.c_void_p(16)
    return lib.resispec_verify_ex(p, p, p, p, ctypes.c_float(T), 0, p, p, dims,
                                  ctypes.byref(opts) if opts else None, None)


def test_synchronous_argument_errors(lib):
    D = rs.Dims
    assert _call(lib, D(1, 2, 10, 1, rs.F32), T=0.0) == rs.E_ARG
    assert _call(lib, D(1, 2, 10, 1, rs.F32), T=-1.0) == rs.E_ARG
    assert _call(lib, D(1, 2, 10, 1, rs.F32), T=float("nan")) == rs.E_ARG
    assert _call(lib, D(1, 2, 10, 1, rs.F32), T=float("inf")) == rs.E_ARG
    assert _call(lib, D(1, 2, 0, 1, rs.F32)) == rs.E_SHAPE
    assert _call(lib, D(1, 2, rs.MAX_VOCAB + 1, 1, rs.F32)) == rs.E_SHAPE
    assert _call(lib, D(-1, 2, 10, 1, rs.F32)) == rs.E_SHAPE
    assert _call(lib, D(1, rs.MAX_NODES + 1, 10, 1, rs.F32)) == rs.E_SHAPE
    assert _call(lib, D(1, 2, 10, 3, rs.F32)) == rs.E_SHAPE      # depth > nodes
    assert _call(lib, D(1, 2, 10, 1, 7)) == rs.E_DTYPE
    assert _call(lib, D(1, 2, 10, 1, rs.F32), null=True) == rs.E_ARG
    assert _call(lib, D(0, 2, 10, 1, rs.F32), null=True) == rs.E_OK   # empty batch: no launch


def test_plan_without_device(lib):
    # the bench workload (B = 64, V = 151936 fp32, a binary tree) cannot sit
    # on chip at once: the automatic choice streams it, with 256-thread CTAs
    # (about two children per node) in clusters of 6 (one wave of 76 on 456
    # CTA slots: the tree is 5 levels deep)
    p = rs.plan(64, 62, 151936, 5, "f32")
    assert p["kernel_name"] == "stream" and p["cluster_size"] == 6
    assert p["block_threads"] == 256
    assert p["smem_bytes"] <= 228 * 1024 // 3 - 1024   # three CTAs per SM
    assert p["slice_elems"] % 8 == 0 and p["slice_elems"] * 6 >= 151936
    # 512-thread CTAs for wider trees and for batches that fit clusters of 16
    assert rs.plan(1, 62, 151936, 5, "f32")["block_threads"] == 512
    assert rs.plan(128, 16, 256000, 1, "bf16")["block_threads"] == 512
    p4 = rs.plan(128, 4, 256000, 1, "bf16")   # single position, k = 4
    assert (p4["cluster_size"], p4["block_threads"]) == (6, 256)
    # shallow trees accept more waves: 128 single-position sequences in
    # clusters of 8; deep trees of 32 sequences in clusters of 8 (one wave);
    # of 128 sequences, whose one-wave slices would be too long, in clusters
    # of 4 (two waves)
    assert rs.plan(128, 16, 256000, 1, "bf16", kernel="stream")["cluster_size"] == 8
    assert rs.plan(32, 488, 256000, 6, "bf16", kernel="stream")["cluster_size"] == 8
    assert rs.plan(128, 488, 256000, 6, "bf16", kernel="stream")["cluster_size"] == 4
    # an explicit block size is kept
    p = rs.plan(64, 62, 151936, 5, "f32", block_threads=512)
    assert p["block_threads"] == 512 and p["cluster_size"] == 4
    # the streaming kernel moves 16-byte vectors with per-thread asynchronous
    # copies, not bulk (TMA) copies; the resident kernel uses bulk copies
    assert p["uses_tma"] == 0 and p["vector_loads"] == 1
    r = rs.plan(64, 62, 151936, 5, "f32", kernel="resident")
    assert r["uses_tma"] == 1 and r["vector_loads"] == 1
    for B in (1, 7, 64, 128, 1000):
        p = rs.plan(B, 488, 256000, 6, "bf16", kernel="stream")
        assert p["smem_bytes"] <= 228 * 1024 // 2 - 1024
    p = rs.plan(64, 62, 151936, 5, "f32", kernel="resident")
    assert p["kernel_name"] == "resident" and p["cluster_size"] in (8, 16)
    assert p["slice_elems"] * p["cluster_size"] >= 151936
    assert p["smem_bytes"] <= 227 * 1024
    # the automatic choice is the streaming kernel, also for a batch that
    # would fit on chip; the resident kernel runs when asked for
    assert rs.plan(1, 60, 32000, 5, "bf16")["kernel_name"] == "stream"
    assert rs.plan(1, 60, 32000, 5, "bf16", kernel="resident")["kernel_name"] == "resident"
    p = rs.plan(1, 12, 64, 4, "f32", cluster_size=1)
    assert p["cluster_size"] == 1 and p["slice_elems"] == 64
    p = rs.plan(1, 12, 61, 4, "f32", cluster_size=2)
    assert p["uses_tma"] == 0 and p["vector_loads"] == 0   # 61 * 4 bytes per row: not aligned
    p = rs.plan(1, 12, 64, 4, "bf16", no_tma=True)
    assert p["uses_tma"] == 0
    for V in (1, 7, 32000, 128256, 256000, rs.MAX_VOCAB):
        for kernel in ("resident", "stream"):
            p = rs.plan(128, 488, V, 6, "bf16", kernel=kernel)
            assert p["smem_bytes"] <= 227 * 1024
    # streaming: the largest cluster size within the wave bound
    assert rs.plan(16, 32, 128256, 4, "bf16", kernel="stream")["cluster_size"] == 16
    # the streaming kernel holds no rows: one CTA per sequence at any V
    p = rs.plan(1, 2, rs.MAX_VOCAB, 1, "f32", cluster_size=1, kernel="stream")
    assert p["cluster_size"] == 1 and p["slice_elems"] == rs.MAX_VOCAB
    p = rs.plan(1, 2, 1000, 1, "f32", cluster_size=3)   # any cluster size up to 16
    assert p["cluster_size"] == 3 and p["slice_elems"] * 3 >= 1000
    with pytest.raises(rs.ResispecError):
        rs.plan(1, 2, 10, 1, "f32", cluster_size=17)
    with pytest.raises(rs.ResispecError):
        rs.plan(1, 2, rs.MAX_VOCAB, 1, "f32", cluster_size=1, kernel="resident")  # 2 MB on one CTA
    o = rs.make_opts(kernel="stream")
    o.flags |= rs.FLAG_RESIDENT                   # both kernels forced: argument error
    assert lib.resispec_plan(rs.Dims(1, 2, 10, 1, rs.F32), o, None) == rs.E_ARG
    # SpecInfer runs on the streaming kernel only (its residual is evaluated
    # from the raw logits, which the resident kernel does not keep)
    assert rs.plan(1, 60, 32000, 5, "bf16", mode=rs.MODE_SPECINFER)["kernel_name"] == "stream"
    o = rs.make_opts(mode=rs.MODE_SPECINFER, kernel="resident")
    assert lib.resispec_plan(rs.Dims(1, 60, 32000, 5, rs.BF16), o, None) == rs.E_ARG
    # the variants run on the streaming kernel only
    for kw in (dict(z_rule=rs.Z_RULE_APPLIED), dict(proxy_denominator=True),
               dict(fill=rs.FILL_LEVEL)):
        assert rs.plan(1, 2, 64, 1, "f32", **kw)["kernel_name"] == "stream"
        o = rs.make_opts(**kw)
        o.flags |= rs.FLAG_RESIDENT
        assert lib.resispec_plan(rs.Dims(1, 2, 64, 1, rs.F32), o, None) == rs.E_ARG


def test_no_cpu_path():
    torch = pytest.importorskip("torch")
    t = torch.zeros((1, 2, 8))
    with pytest.raises(ValueError):
        rs.verify(t, t, torch.zeros(1, dtype=torch.int32), torch.zeros((1, 1), dtype=torch.int32),
                  1.0, 0, max_depth=1)


def test_binding_constants_match_the_header():
    """Every RESISPEC_* constant the header defines has the same value in the
    Python binding (flags, status bits, phases, limits, kernels, ABI)."""
    text = open(HEADER).read()
    defs = dict((n, int(v)) for n, v in re.findall(r"^#define (RESISPEC_[A-Z0-9_]+) (\d+)", text,
                                                   flags=re.M))
    assert len(defs) >= 25
    phase = {"SETUP": "setup", "NORM": "norm", "NORM_X": "norm_exchange", "TEST": "test",
             "REJECT": "reject", "DRAW": "draw"}
    for name, value in defs.items():
        short = name[len("RESISPEC_"):]
        if short == "PHASES":
            assert len(rs.PHASES) == value
        elif short.startswith("PHASE_"):
            assert rs.PHASES.index(phase[short[len("PHASE_"):]]) == value, name
        elif short == "ABI_VERSION":
            assert rs.load_library().resispec_abi_version() == value
        else:
            assert hasattr(rs, short), f"binding lacks {short}"
            assert getattr(rs, short) == value, name


def test_header_is_c_and_library_links_from_c(tmp_path, lib):
    """include/resispec.h compiles as C11 and a C program links against the
    library and calls it (no device work: the ABI version and a synchronous
    argument error)."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "c_abi.c"
    src.write_text(r'''
#include <stdio.h>
#include <stdint.h>
#include "resispec.h"
int main(void) {
  resispec_opts o;
  resispec_opts_default(&o);
  resispec_dims d = {1, 2, 10, 1, RESISPEC_F32};
  int rc = resispec_verify_ex(0, 0, 0, 0, 1.0f, 0, 0, 0, d, &o, 0);
  printf("%d %d %d\n", resispec_abi_version(), rc == RESISPEC_E_ARG, o.seq_stride == -1);
  return 0;
}
''')
    libdir = os.path.dirname(rs._build.LIB)
    exe = tmp_path / "c_abi"
    subprocess.run([gcc, "-std=c11", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"),
                    str(src), "-o", str(exe), "-L", libdir, "-lresispec",
                    f"-Wl,-rpath,{libdir}"], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()
    assert out == ["4", "1", "1"]


@pytest.mark.gpu
def test_c_program_verifies_a_batch_on_the_device(tmp_path, lib):
    """A C program (no Python on its path) allocates device buffers with the
    CUDA runtime, copies a batch in, calls resispec_verify and copies the
    accepted tokens and accept lengths back; they match the fp64 oracle on
    every sequence away from a near tie."""
    import shutil
    import subprocess
    import oracle
    from paper_2608_24411_gb300 import workloads as W
    gcc = shutil.which("gcc")
    cuda = "/usr/local/cuda"
    if gcc is None or not os.path.exists(os.path.join(cuda, "include", "cuda_runtime_api.h")):
        pytest.skip("no C compiler or CUDA headers")
    w = W.WORKLOADS["tiny-chain-v64"]
    B = 512
    inp = W.make_inputs_np(w, seed=21, batch=B)
    N, V, D = w.num_nodes, w.vocab, w.max_depth
    seed = 2024
    src = tmp_path / "c_verify.c"
    src.write_text(r'''
#include <stdio.h>
#include <stdlib.h>
#include <stdint.h>
#include <cuda_runtime_api.h>
#include "resispec.h"
static void* slurp(const char* path, size_t n) {
  void* p = malloc(n);
  FILE* f = fopen(path, "rb");
  if (!f || fread(p, 1, n, f) != n) { fprintf(stderr, "read %s\n", path); exit(2); }
  fclose(f);
  return p;
}
static void* to_device(const void* h, size_t n) {
  void* d = 0;
  if (cudaMalloc(&d, n) != cudaSuccess || cudaMemcpy(d, h, n, cudaMemcpyHostToDevice) != cudaSuccess) {
    fprintf(stderr, "device copy failed\n"); exit(3);
  }
  return d;
}
int main(int argc, char** argv) {
  const int B = atoi(argv[2]), N = atoi(argv[3]), V = atoi(argv[4]), D = atoi(argv[5]);
  const float T = (float)atof(argv[6]);
  const uint64_t seed = strtoull(argv[7], 0, 10);
  char path[4096];
  const size_t nlog = (size_t)B * (N + 1) * V * sizeof(float);
  snprintf(path, sizeof path, "%s/target.bin", argv[1]);
  void* t = to_device(slurp(path, nlog), nlog);
  snprintf(path, sizeof path, "%s/draft.bin", argv[1]);
  void* d = to_device(slurp(path, nlog), nlog);
  snprintf(path, sizeof path, "%s/parents.bin", argv[1]);
  int32_t* par = (int32_t*)to_device(slurp(path, N * 4), N * 4);
  snprintf(path, sizeof path, "%s/cand.bin", argv[1]);
  int32_t* cand = (int32_t*)to_device(slurp(path, (size_t)B * N * 4), (size_t)B * N * 4);
  int32_t *tok = 0, *len = 0;
  cudaMalloc((void**)&tok, (size_t)B * (D + 1) * 4);
  cudaMalloc((void**)&len, (size_t)B * 4);
  resispec_dims dims = {B, N, V, D, RESISPEC_F32};
  int rc = resispec_verify(t, d, par, cand, T, seed, tok, len, dims, 0);
  if (rc != RESISPEC_OK) { fprintf(stderr, "verify: %s\n", resispec_status_string(rc)); return 4; }
  if (cudaDeviceSynchronize() != cudaSuccess) { fprintf(stderr, "sync failed\n"); return 5; }
  int32_t* htok = (int32_t*)malloc((size_t)B * (D + 1) * 4);
  int32_t* hlen = (int32_t*)malloc((size_t)B * 4);
  cudaMemcpy(htok, tok, (size_t)B * (D + 1) * 4, cudaMemcpyDeviceToHost);
  cudaMemcpy(hlen, len, (size_t)B * 4, cudaMemcpyDeviceToHost);
  snprintf(path, sizeof path, "%s/out.bin", argv[1]);
  FILE* f = fopen(path, "wb");
  fwrite(htok, 4, (size_t)B * (D + 1), f);
  fwrite(hlen, 4, (size_t)B, f);
  fclose(f);
  cudaFree(t); cudaFree(d); cudaFree(par); cudaFree(cand); cudaFree(tok); cudaFree(len);
  return 0;
}
''')
    for name in ("target", "draft"):
        np.ascontiguousarray(inp[name], np.float32).tofile(tmp_path / f"{name}.bin")
    np.ascontiguousarray(inp["parents"], np.int32).tofile(tmp_path / "parents.bin")
    np.ascontiguousarray(inp["cand"], np.int32).tofile(tmp_path / "cand.bin")
    libdir = os.path.dirname(rs._build.LIB)
    cudalib = next((p for p in (os.path.join(cuda, "lib64"), os.path.join(cuda, "lib"))
                    if os.path.exists(p)), os.path.join(cuda, "lib64"))
    exe = tmp_path / "c_verify"
    subprocess.run([gcc, "-std=c11", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"),
                    "-I", os.path.join(cuda, "include"), str(src), "-o", str(exe),
                    "-L", libdir, "-lresispec", "-L", cudalib, "-lcudart",
                    f"-Wl,-rpath,{libdir}", f"-Wl,-rpath,{cudalib}"], check=True)
    subprocess.run([str(exe), str(tmp_path), str(B), str(N), str(V), str(D), repr(w.temperature),
                    str(seed)], check=True, timeout=120)
    out = np.fromfile(tmp_path / "out.bin", dtype=np.int32)
    toks, alen = out[: B * (D + 1)].reshape(B, D + 1), out[B * (D + 1):]
    o = oracle.verify(inp["target"], inp["draft"], inp["parents"], inp["cand"], w.temperature,
                      seed, max_depth=D)
    clean = (o["accept_margin"] > 1e-5) & (o["sample_margin"] > 1e-6)
    assert clean.sum() >= 0.99 * B
    np.testing.assert_array_equal(alen[clean], o["accept_len"][clean])
    np.testing.assert_array_equal(toks[clean], o["tokens"][clean])


@pytest.mark.gpu
def test_graft_entry_smoke():
    """The round-end smoke entry point: small calls on cuda:0 in every mode
    and kernel it supports, checked against the oracle."""
    import __graft_entry__
    __graft_entry__.smoke()
