"""fp64 CPU oracle of the ResiSpec verification walk.

TEST INFRASTRUCTURE ONLY: ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` are the only callers.  The
product path (``paper_2608_24411_gb300``) never imports this package and
fails loudly when its CUDA library is missing.

Two independent pieces live here:

* ``resispec_oracle.c`` (wrapped below): the literal walk of Algorithm 1 /
  GetProxy / Eq. 2 (Sec. 3) over a draft tree, fp64, threaded over sequences.
* ``enumerator.py``: an exact enumerator of the output distribution of the
  same rules for tiny vocabularies (numpy, no sampling), used to pin the C
  oracle.

Parity status of each function is stated in ``resispec_oracle.c``; the
deficit split of GetProxy (reading R2) is "parity unpinned" beyond the
hand-worked example and Theorem 2's L1 closed form.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "resispec_oracle.c")
# tolerance machinery for proxy-denominator rows, kept apart from the walk
_SRC_ERR = os.path.join(_HERE, "fp32_error_bound.c")
_SOURCES = (_SRC, _SRC_ERR, os.path.join(_HERE, "fp32_error_bound.h"))
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIBDIR, "libresispec_oracle.so")

MODE_RESISPEC = 0
MODE_SPECINFER = 1
F32 = 0
BF16 = 1
FILL_CAPACITY = 0  # the deficit in proportion to the remaining capacity (R2)
FILL_LEVEL = 1     # r = min(lam q, p) at a common level lam (R10)

ERR_TREE = 1
ERR_TOKEN = 2
ERR_NONFINITE = 4
ERR_EMPTY_ROW = 8
ERR_DEPTH = 16
INFO_DEGENERATE = 256

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no -ffast-math, no FMA contraction)."""
    os.makedirs(_LIBDIR, exist_ok=True)
    if (not force and os.path.exists(_LIB)
            and all(os.path.getmtime(_LIB) >= os.path.getmtime(f) for f in _SOURCES)):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread",
           "-ffp-contract=off", "-fno-fast-math", "-o", tmp, _SRC, _SRC_ERR, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


class _Args(ctypes.Structure):
    _fields_ = [
        ("B", ctypes.c_int32), ("N", ctypes.c_int32), ("V", ctypes.c_int32),
        ("D", ctypes.c_int32), ("dtype", ctypes.c_int32), ("mode", ctypes.c_int32),
        ("decide_fp64", ctypes.c_int32), ("check_invariants", ctypes.c_int32),
        ("nthreads", ctypes.c_int32), ("pad_", ctypes.c_int32),
        ("seq_stride", ctypes.c_int64),
        ("target", ctypes.c_void_p), ("draft", ctypes.c_void_p),
        ("parents", ctypes.c_void_p), ("cand", ctypes.c_void_p),
        ("seq_ids", ctypes.c_void_p),
        ("temperature", ctypes.c_double), ("seed", ctypes.c_uint64),
        ("out_tokens", ctypes.c_void_p), ("out_len", ctypes.c_void_p),
        ("out_nodes", ctypes.c_void_p), ("out_dist", ctypes.c_void_p),
        ("out_accept_margin", ctypes.c_void_p), ("out_sample_margin", ctypes.c_void_p),
        ("out_status", ctypes.c_void_p), ("out_rejects", ctypes.c_void_p),
        ("out_rows", ctypes.c_void_p), ("out_inv_err", ctypes.c_void_p),
        ("out_cond", ctypes.c_void_p), ("parents_stride", ctypes.c_int64),
        ("z_rule", ctypes.c_int32), ("denom_update", ctypes.c_int32),
        ("draft_out", ctypes.c_void_p), ("out_draft_margin", ctypes.c_void_p),
        ("fill", ctypes.c_int32), ("pad2_", ctypes.c_int32),
        ("out_dist_err", ctypes.c_void_p),
    ]


def load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            lib.oracle_verify.argtypes = [ctypes.POINTER(_Args)]
            lib.oracle_verify.restype = ctypes.c_int
            lib.oracle_uniform.argtypes = [ctypes.c_uint64, ctypes.c_int64,
                                           ctypes.c_int64, ctypes.c_int]
            lib.oracle_uniform.restype = ctypes.c_double
            lib.oracle_philox4x64_10.argtypes = [ctypes.c_void_p, ctypes.c_void_p,
                                                 ctypes.c_void_p]
            lib.oracle_philox4x64_10.restype = None
            lib.oracle_softmax.argtypes = [ctypes.c_void_p, ctypes.c_int,
                                           ctypes.c_double, ctypes.c_void_p]
            lib.oracle_softmax.restype = ctypes.c_int
            lib.oracle_get_proxy.argtypes = [ctypes.c_void_p, ctypes.c_void_p,
                                             ctypes.c_int, ctypes.c_int,
                                             ctypes.c_void_p, ctypes.c_void_p]
            lib.oracle_get_proxy.restype = ctypes.c_double
            lib.oracle_get_proxy_z.argtypes = [ctypes.c_void_p, ctypes.c_void_p,
                                               ctypes.c_int, ctypes.c_int, ctypes.c_double,
                                               ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p]
            lib.oracle_get_proxy_z.restype = ctypes.c_double
            lib.oracle_reject.argtypes = [ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p,
                                          ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                          ctypes.c_void_p, ctypes.c_void_p,
                                          ctypes.c_void_p]
            lib.oracle_reject.restype = ctypes.c_int
            lib.oracle_reject_z.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                            ctypes.c_void_p,
                                            ctypes.c_void_p, ctypes.c_int, ctypes.c_int,
                                            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                            ctypes.c_void_p, ctypes.c_void_p]
            lib.oracle_reject_z.restype = ctypes.c_int
            lib.oracle_budget.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                                          ctypes.c_int, ctypes.c_int]
            lib.oracle_budget.restype = ctypes.c_double
            lib.oracle_sample.argtypes = [ctypes.c_void_p, ctypes.c_int,
                                          ctypes.c_double, ctypes.c_void_p]
            lib.oracle_sample.restype = ctypes.c_int
            lib.oracle_fp32err_init.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p]
            lib.oracle_fp32err_init.restype = None
            lib.oracle_fp32err_reject.argtypes = [ctypes.c_void_p] * 4 + [
                ctypes.c_int, ctypes.c_int, ctypes.c_double, ctypes.c_double, ctypes.c_double,
                ctypes.c_void_p, ctypes.c_void_p]
            lib.oracle_fp32err_reject.restype = None
            lib.oracle_args_size.restype = ctypes.c_int
            if lib.oracle_args_size() != ctypes.sizeof(_Args):
                raise RuntimeError("oracle_args layout mismatch")
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


# ---------------------------------------------------------------- primitives
def philox4x64_10(counter, key):
    """Raw Philox4x64-10 block (4 uint64 words)."""
    lib = load()
    c = np.ascontiguousarray(counter, dtype=np.uint64)
    k = np.ascontiguousarray(key, dtype=np.uint64)
    out = np.zeros(4, dtype=np.uint64)
    lib.oracle_philox4x64_10(c.ctypes.data, k.ctypes.data, out.ctypes.data)
    return out


def uniform(seed: int, seq: int, row: int, draw: int) -> float:
    return load().oracle_uniform(seed, seq, row, draw)


def softmax(z, temperature: float):
    """Tempered softmax of one row; returns (p, status)."""
    z = _f64(z)
    p = np.zeros_like(z)
    st = load().oracle_softmax(z.ctypes.data, z.size, float(temperature), p.ctypes.data)
    return p, st


def get_proxy(p, q, x0: int, fill: int = FILL_CAPACITY, Z=None):
    """GetProxy(p, q, x0) -> (k, r, Z).  ``fill``: FILL_CAPACITY (the deficit
    in proportion to the capacity p - r) or FILL_LEVEL (r = min(lam q, p) at
    the level lam that meets the budget); ``Z``: the budget (default
    q(x0) - p(x0), Algorithm 1)."""
    p, q = _f64(p), _f64(q)
    k, r = np.zeros_like(p), np.zeros_like(p)
    if Z is None:
        Z = q[int(x0)] - p[int(x0)]
    Z = load().oracle_get_proxy_z(p.ctypes.data, q.ctypes.data, p.size, int(x0), float(Z),
                                  int(fill), k.ctypes.data, r.ctypes.data)
    return k, r, Z


def budget(R, q, x0: int, z_rule: int = 0) -> float:
    """The ResiSpec budget of a rejection of x0: z_rule 0 = Algorithm 1
    (q(x0) - R(x0)), 1 = Z_applied (max(Z*, |gap|) clamped to 1 - R(x0))."""
    R, q = _f64(R), _f64(q)
    return load().oracle_budget(R.ctypes.data, q.ctypes.data, R.size, int(x0), int(z_rule))


def reject(mode: int, R, q, x0: int, check: bool = True, z_rule: int = 0,
           fill: int = FILL_CAPACITY):
    """One rejection of x0: returns (R', changed, invariant_error)."""
    R = _f64(R).copy()
    q = _f64(q)
    V = R.size
    K, r, tmp = np.zeros(V), np.zeros(V), np.zeros(V)
    err = np.zeros(1)
    changed = load().oracle_reject_z(int(mode), int(z_rule), int(fill), R.ctypes.data,
                                     q.ctypes.data, V,
                                     int(x0), K.ctypes.data, r.ctypes.data, tmp.ctypes.data,
                                     err.ctypes.data if check else None, None)
    return R, bool(changed), float(err[0])


def fp32_error_init(v):
    """Bounds of the rounding of fp32 tempered softmax values v (tolerance
    machinery of proxy-denominator rows, ``fp32_error_bound.c``)."""
    v = _f64(v)
    e = np.zeros_like(v)
    load().oracle_fp32err_init(v.ctypes.data, v.size, e.ctypes.data)
    return e


def fp32_error_reject(R, D, r, K, x0, Z, level, mu, eR, eD):
    """One rejection's propagation of the bounds (eR, eD) of R and D
    (``fp32_error_bound.c``); returns the bounds of R' = r / sum r and D' = K."""
    R, D, r, K = _f64(R), _f64(D), _f64(r), _f64(K)
    eR, eD = _f64(eR).copy(), _f64(eD).copy()
    load().oracle_fp32err_reject(R.ctypes.data, D.ctypes.data, r.ctypes.data, K.ctypes.data,
                                 R.size, int(x0), float(Z), float(level), float(mu),
                                 eR.ctypes.data, eD.ctypes.data)
    return eR, eD


def sample(R, u: float):
    """Inverse-CDF draw -> (token, relative margin)."""
    R = _f64(R)
    m = np.zeros(1)
    x = load().oracle_sample(R.ctypes.data, R.size, float(u), m.ctypes.data)
    return x, float(m[0])


# ---------------------------------------------------------------- full walk
def verify(target, draft, parents, cand, temperature, seed, *, mode=MODE_RESISPEC,
           max_depth=None, seq_stride=None, seq_ids=None, nthreads=None,
           check_invariants=False, decide_fp64=True, want_dist=False, z_rule=0,
           denom_update=False, draft_children=False, fill=0, want_dist_err=False):
    """Run the oracle walk.

    ``target``/``draft``: float32 arrays, or uint16 arrays holding bf16 bit
    patterns, shaped [B, N+1, V] (or [N+1, V] with ``seq_stride=0`` to share
    one set of rows across all B sequences, in which case ``cand`` gives B).
    ``parents``: int32 [N] (one tree for every sequence) or [B, N] (a tree
    per sequence); ``cand``: int32 [B, N].
    ``decide_fp64``: every accept test is the paper's u < R(x)/D(x) in fp64
    (Algorithm 1); False takes it as u * D(x) < R(x) on values rounded to
    fp32, a diagnostic of how a single-precision evaluation decides.
    ``want_dist_err``: also return "dist_err" [B, V], a first-order bound of
    the error of an fp32 evaluation of "dist" for rows whose test
    denominator is the proxy (``denom_update``; reading R11), 0 elsewhere.
    Returns a dict of numpy arrays.
    """
    lib = load()
    if target.dtype == np.uint16:
        dtype = BF16
    elif target.dtype == np.float32:
        dtype = F32
    else:
        raise TypeError("target must be float32 or uint16 (bf16 bits)")
    if draft.dtype != target.dtype or draft.shape != target.shape:
        raise TypeError("draft must match target")
    target = np.ascontiguousarray(target)
    draft = np.ascontiguousarray(draft)
    parents = np.ascontiguousarray(parents, dtype=np.int32)
    cand = np.ascontiguousarray(cand, dtype=np.int32)
    per_seq = parents.ndim == 2
    N = parents.shape[-1] if per_seq else parents.size
    B = cand.shape[0] if cand.ndim == 2 else (target.shape[0] if target.ndim == 3 else 1)
    if cand.ndim != 2:
        cand = cand.reshape(B, N)
    V = target.shape[-1]
    if seq_stride is None:
        seq_stride = (N + 1) * V
    if per_seq and parents.shape[0] != B:
        raise ValueError("per-sequence parents must be [B, N]")
    if max_depth is None:
        max_depth = max((tree_depth(t) for t in parents), default=0) if per_seq \
            else tree_depth(parents)
    D = int(max_depth)
    if seq_ids is not None:
        seq_ids = np.ascontiguousarray(seq_ids, dtype=np.int32)
    out = {
        "tokens": np.full((B, D + 1), -1, np.int32),
        "accept_len": np.zeros(B, np.int32),
        "nodes": np.full((B, max(D, 1)), -1, np.int32),
        "accept_margin": np.zeros(B),
        "sample_margin": np.zeros(B),
        "status": np.zeros(B, np.int32),
        "rejects": np.zeros(B, np.int32),
        "rows": np.zeros(B, np.int32),
        "inv_err": np.zeros(B),
        "cond": np.ones(B),
    }
    if want_dist:
        out["dist"] = np.zeros((B, V))
    if want_dist_err:
        out["dist_err"] = np.zeros((B, V))
    a = _Args()
    a.B, a.N, a.V, a.D = B, N, V, D
    a.dtype, a.mode = dtype, int(mode)
    a.decide_fp64 = int(bool(decide_fp64))
    a.check_invariants = int(bool(check_invariants))
    a.nthreads = int(nthreads or os.cpu_count() or 1)
    a.seq_stride = int(seq_stride)
    a.target, a.draft = target.ctypes.data, draft.ctypes.data
    a.parents, a.cand = parents.ctypes.data, cand.ctypes.data
    a.parents_stride = N if per_seq else 0
    a.z_rule = int(z_rule)
    a.denom_update = int(bool(denom_update))
    a.fill = int(fill)
    if draft_children:  # candidates drawn from each visited node's q (cand is ignored)
        out["drafted"] = np.full((B, N), -1, np.int32)
        out["draft_margin"] = np.zeros(B)
        a.draft_out = out["drafted"].ctypes.data
        a.out_draft_margin = out["draft_margin"].ctypes.data
    a.seq_ids = _ptr(seq_ids)
    a.temperature = float(np.float32(temperature))
    a.seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    a.out_tokens = out["tokens"].ctypes.data
    a.out_len = out["accept_len"].ctypes.data
    a.out_nodes = out["nodes"].ctypes.data
    a.out_dist = out["dist"].ctypes.data if want_dist else None
    a.out_dist_err = out["dist_err"].ctypes.data if want_dist_err else None
    a.out_accept_margin = out["accept_margin"].ctypes.data
    a.out_sample_margin = out["sample_margin"].ctypes.data
    a.out_status = out["status"].ctypes.data
    a.out_rejects = out["rejects"].ctypes.data
    a.out_rows = out["rows"].ctypes.data
    a.out_inv_err = out["inv_err"].ctypes.data
    a.out_cond = out["cond"].ctypes.data
    rc = lib.oracle_verify(ctypes.byref(a))
    if rc != 0:
        raise ValueError("oracle_verify rejected its arguments")
    if D == 0:
        out["nodes"] = out["nodes"][:, :0]
    return out


def tree_depth(parents) -> int:
    """Depth (number of edges from the root) of the deepest node."""
    parents = np.asarray(parents)
    depth = np.zeros(parents.size, dtype=np.int64)
    for c, p in enumerate(parents):
        depth[c] = 1 if p < 0 else depth[p] + 1
    return int(depth.max()) if parents.size else 0
