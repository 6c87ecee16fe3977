"""The C ABI without a GPU: the library builds and loads, exports every
function include/resispec.h declares, and rejects bad arguments
synchronously (before any device work)."""
import ctypes
import os
import re

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
    assert lib.resispec_abi_version() == 3


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
    # the bench workload (B = 64, V = 151936 fp32) cannot sit on chip at once:
    # the automatic choice streams it, in clusters of 4 CTAs (one wave: the
    # tree is 5 levels deep)
    p = rs.plan(64, 62, 151936, 5, "f32")
    assert p["kernel_name"] == "stream" and p["cluster_size"] == 4
    assert p["smem_bytes"] <= 228 * 1024 // 2 - 1024   # two CTAs per SM
    assert p["slice_elems"] % 8 == 0 and p["slice_elems"] * 4 >= 151936
    # shallow trees accept more waves: 128 single-position sequences in
    # clusters of 8; deep trees of 32 sequences in clusters of 8 (one wave)
    assert rs.plan(128, 16, 256000, 1, "bf16", kernel="stream")["cluster_size"] == 8
    assert rs.plan(32, 488, 256000, 6, "bf16", kernel="stream")["cluster_size"] == 8
    assert p["uses_tma"] == 1
    for B in (1, 7, 64, 128, 1000):
        p = rs.plan(B, 488, 256000, 6, "bf16", kernel="stream")
        assert p["smem_bytes"] <= 228 * 1024 // 2 - 1024
    p = rs.plan(64, 62, 151936, 5, "f32", kernel="resident")
    assert p["kernel_name"] == "resident" and p["cluster_size"] in (8, 16)
    assert p["slice_elems"] * p["cluster_size"] >= 151936
    assert p["smem_bytes"] <= 227 * 1024
    # a small batch that fits on chip stays resident
    p = rs.plan(1, 60, 32000, 5, "bf16")
    assert p["kernel_name"] == "resident"
    p = rs.plan(1, 12, 64, 4, "f32", cluster_size=1)
    assert p["cluster_size"] == 1 and p["slice_elems"] == 64
    p = rs.plan(1, 12, 61, 4, "f32", cluster_size=2)
    assert p["uses_tma"] == 0                      # 61 * 4 bytes per row: not 16-byte aligned
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
    assert out == ["3", "1", "1"]
