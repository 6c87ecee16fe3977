"""GB300-native verification hot path of ResiSpec multi-candidate speculative
sampling.

Python binding of the C ABI in ``include/resispec.h``: argument marshalling
only.  Every step of the verification (tempered normaliser, accept tests,
residual shaping, tree walk, residual / bonus sampling, Philox) runs in the
sm_103a CUDA library ``_lib/libresispec.so``.  There is no CPU path: calls
raise when the library is missing or a tensor is not on a CUDA device.

Inputs follow the paper's statement of the verification problem (Sec. 3,
Algorithm 1): per sequence, target and draft logits for the root and every
draft-tree node ([B, N+1, V], row 0 = root, row j+1 = node j), the tree as
parent indices, and the candidate token proposed at each node.
"""
from __future__ import annotations

import ctypes
import os
import threading

from . import _build

MODE_RESISPEC = 0
MODE_SPECINFER = 1
F32 = 0
BF16 = 1

ERR_TREE = 1
ERR_TOKEN = 2
ERR_NONFINITE = 4
ERR_EMPTY_ROW = 8
ERR_DEPTH = 16
ERR_TIMEOUT = 32
ERR_FANOUT = 64
INFO_DEGENERATE = 256
FLAG_NO_TMA = 1
FLAG_PREFETCH = 2
FLAG_RESIDENT = 4
FLAG_STREAM = 8
FLAG_Z_APPLIED = 16
FLAG_PROXY_DENOM = 32
FLAG_LEVEL_FILL = 64
Z_RULE_ALG1 = 0       # ResiSpec budget Z = q(x0) - R(x0) (Algorithm 1)
Z_RULE_APPLIED = 1    # Z = max(Z*, |gap|) clamped to 1 - R(x0) (Sec. 5.3 heuristic)
FILL_CAPACITY = 0     # GetProxy's deficit in proportion to the capacity R - r (default)
FILL_LEVEL = 1        # r = min(lam q, R) at the level lam that meets the budget
PHASES = ("setup", "norm", "norm_exchange", "test", "reject", "draw")
KERNEL_RESIDENT = 0
KERNEL_STREAM = 1
KERNELS = {"auto": None, "resident": KERNEL_RESIDENT, "stream": KERNEL_STREAM}

MAX_VOCAB = 262144
MAX_NODES = 4096
MAX_FANOUT_STREAM = 128

E_OK, E_ARG, E_SHAPE, E_DTYPE, E_UNSUPPORTED, E_CUDA = range(6)

_lock = threading.Lock()
_lib = None

EXPORTED = (
    "resispec_opts_default", "resispec_verify", "resispec_verify_ex", "resispec_plan",
    "resispec_uniforms", "resispec_status_string", "resispec_last_error",
    "resispec_abi_version",
)


class Dims(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("num_nodes", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("max_depth", ctypes.c_int32),
                ("dtype", ctypes.c_int32)]


class Opts(ctypes.Structure):
    _fields_ = [("mode", ctypes.c_int32), ("cluster_size", ctypes.c_int32),
                ("block_threads", ctypes.c_int32), ("flags", ctypes.c_int32),
                ("seq_stride", ctypes.c_int64), ("status", ctypes.c_void_p),
                ("out_nodes", ctypes.c_void_p), ("out_dist", ctypes.c_void_p),
                ("out_rejects", ctypes.c_void_p), ("out_phase_cycles", ctypes.c_void_p),
                ("out_candidates", ctypes.c_void_p),
                ("parents_stride", ctypes.c_int64)]


class PlanInfo(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "kernel", "cluster_size", "block_threads", "smem_bytes", "slice_elems", "uses_tma",
        "vector_loads", "active_clusters")]


class ResispecError(RuntimeError):
    def __init__(self, code: int, where: str):
        lib = _lib
        msg = lib.resispec_status_string(code).decode() if lib else str(code)
        extra = lib.resispec_last_error().decode() if lib else ""
        super().__init__(f"{where}: {msg}" + (f" ({extra})" if extra else ""))
        self.code = code


def build(force: bool = False) -> str:
    """Compile the CUDA library in-tree for sm_103a."""
    return _build.build(force=force)


def library_path() -> str:
    return _build.LIB


def load_library():
    """Load the built library; raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(_build.LIB):
            raise RuntimeError(
                f"CUDA library {_build.LIB} is missing: build it with "
                "paper_2608_24411_gb300.build() (no CPU fallback exists)")
        lib = ctypes.CDLL(_build.LIB)
        vp, i32, i64, u64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64
        lib.resispec_opts_default.argtypes = [ctypes.POINTER(Opts)]
        lib.resispec_opts_default.restype = None
        lib.resispec_verify.argtypes = [vp, vp, vp, vp, ctypes.c_float, u64, vp, vp, Dims, vp]
        lib.resispec_verify.restype = ctypes.c_int
        lib.resispec_verify_ex.argtypes = [vp, vp, vp, vp, ctypes.c_float, u64, vp, vp, Dims,
                                           ctypes.POINTER(Opts), vp]
        lib.resispec_verify_ex.restype = ctypes.c_int
        lib.resispec_plan.argtypes = [Dims, ctypes.POINTER(Opts), ctypes.POINTER(PlanInfo)]
        lib.resispec_plan.restype = ctypes.c_int
        lib.resispec_uniforms.argtypes = [u64, vp, vp, i32, vp, vp, vp]
        lib.resispec_uniforms.restype = ctypes.c_int
        lib.resispec_status_string.argtypes = [ctypes.c_int]
        lib.resispec_status_string.restype = ctypes.c_char_p
        lib.resispec_last_error.argtypes = []
        lib.resispec_last_error.restype = ctypes.c_char_p
        lib.resispec_abi_version.restype = ctypes.c_int
        _lib = lib
        return lib


def _torch():
    import torch
    return torch


def _dtype_code(t) -> int:
    torch = _torch()
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise TypeError(f"logits must be float32 or bfloat16, got {t.dtype}")


def _need_cuda(name, t):
    if t is None:
        return
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor (the library has no CPU path)")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _kernel_flags(kernel) -> int:
    if kernel in (None, "auto"):
        return 0
    k = KERNELS.get(kernel, kernel)
    if k == KERNEL_RESIDENT:
        return FLAG_RESIDENT
    if k == KERNEL_STREAM:
        return FLAG_STREAM
    raise ValueError(f"unknown kernel {kernel!r}")


def make_opts(mode=MODE_RESISPEC, cluster_size=0, block_threads=0, no_tma=False,
              seq_stride=None, status=None, out_nodes=None, out_dist=None,
              out_rejects=None, prefetch=False, kernel=None, z_rule=Z_RULE_ALG1,
              proxy_denominator=False, fill=FILL_CAPACITY) -> Opts:
    lib = load_library()
    o = Opts()
    lib.resispec_opts_default(ctypes.byref(o))
    o.mode = {"resispec": MODE_RESISPEC, "specinfer": MODE_SPECINFER}.get(mode, mode)
    o.cluster_size = int(cluster_size)
    o.block_threads = int(block_threads)
    o.flags = ((FLAG_NO_TMA if no_tma else 0) | (FLAG_PREFETCH if prefetch else 0)
               | _kernel_flags(kernel) | (FLAG_Z_APPLIED if z_rule == Z_RULE_APPLIED else 0)
               | (FLAG_PROXY_DENOM if proxy_denominator else 0)
               | (FLAG_LEVEL_FILL if fill == FILL_LEVEL else 0))
    o.seq_stride = -1 if seq_stride is None else int(seq_stride)
    o.status = None if status is None else status.data_ptr()
    o.out_nodes = None if out_nodes is None else out_nodes.data_ptr()
    o.out_dist = None if out_dist is None else out_dist.data_ptr()
    o.out_rejects = None if out_rejects is None else out_rejects.data_ptr()
    return o


def plan(batch, num_nodes, vocab, max_depth, dtype="f32", **opt_kw) -> dict:
    """Launch shape the library would use for these sizes."""
    lib = load_library()
    d = Dims(int(batch), int(num_nodes), int(vocab), int(max_depth),
             F32 if dtype in ("f32", F32) else BF16)
    o = make_opts(**opt_kw)
    info = PlanInfo()
    rc = lib.resispec_plan(d, ctypes.byref(o), ctypes.byref(info))
    if rc:
        raise ResispecError(rc, "resispec_plan")
    out = {k: getattr(info, k) for k, _ in PlanInfo._fields_}
    out["kernel_name"] = "stream" if info.kernel == KERNEL_STREAM else "resident"
    return out


def verify(target, draft, tree_parents, cand_tokens, temperature, seed, *, max_depth=None,
           mode=MODE_RESISPEC, out_tokens=None, out_accept_len=None, out_nodes=None,
           out_dist=None, out_rejects=None, status=None, cluster_size=0, block_threads=0,
           no_tma=False, seq_stride=None, stream=None, prefetch=False, kernel=None,
           z_rule=Z_RULE_ALG1, proxy_denominator=False, out_phase=None,
           out_candidates=None, fill=FILL_CAPACITY):
    """Verify a batch of draft trees on the GPU.

    target, draft: CUDA tensors [B, N+1, V] (float32 or bfloat16); with
    ``seq_stride=0`` they may be [N+1, V] and are shared by all B sequences.
    tree_parents: int32 CUDA tensor [N] (one tree for every sequence) or
    [B, N] (a tree per sequence); cand_tokens: int32 CUDA tensor [B, N].  Returns (out_tokens [B, D+1], out_accept_len [B]).  Runs on
    ``stream`` (default: torch's current stream) without synchronising.
    ``kernel``: None / "auto" (the library's choice), "resident" or "stream".
    ``z_rule``: the ResiSpec budget, Z_RULE_ALG1 (Algorithm 1) or
    Z_RULE_APPLIED (Sec. 5.3 heuristic; streaming kernel).
    ``proxy_denominator``: after each ResiSpec rejection the accept tests
    and the next GetProxy use that rejection's proxy in place of q (the
    paper's EAGLE integration; streaming kernel).
    ``fill``: how GetProxy fills the deficit, FILL_CAPACITY (in proportion to
    the remaining capacity) or FILL_LEVEL (the draft raised to the level
    that meets the budget; streaming kernel).
    ``out_phase``: optional int64 CUDA tensor [B, len(PHASES)] receiving the
    SM cycles each sequence spent per phase (selects the streaming kernel).
    ``out_candidates``: drafting mode, an int32 CUDA tensor [B, N] that
    receives the children of every visited node drawn from that node's draft
    distribution (then verified); ``cand_tokens`` may be None.
    """
    torch = _torch()
    lib = load_library()
    for name, t in (("target", target), ("draft", draft), ("tree_parents", tree_parents),
                    ("cand_tokens", cand_tokens), ("out_candidates", out_candidates),
                    ("out_tokens", out_tokens),
                    ("out_accept_len", out_accept_len), ("out_nodes", out_nodes),
                    ("out_dist", out_dist), ("out_rejects", out_rejects), ("status", status)):
        _need_cuda(name, t)
    if draft.dtype != target.dtype:
        raise TypeError("target and draft must have the same dtype")
    dt = _dtype_code(target)
    if cand_tokens is None:
        if out_candidates is None:
            raise ValueError("pass cand_tokens, or out_candidates to draft them")
        cand_tokens = out_candidates   # not read in drafting mode; gives B
    if tree_parents.dtype != torch.int32 or cand_tokens.dtype != torch.int32:
        raise TypeError("tree_parents and cand_tokens must be int32")
    per_seq_tree = tree_parents.dim() == 2
    N = int(tree_parents.shape[-1]) if per_seq_tree else int(tree_parents.numel())
    B = int(cand_tokens.shape[0]) if cand_tokens.dim() == 2 else int(target.shape[0])
    if per_seq_tree and int(tree_parents.shape[0]) != B:
        raise ValueError("per-sequence tree_parents must be [B, N]")
    V = int(target.shape[-1])
    if max_depth is None:
        if out_tokens is None:
            raise ValueError("pass max_depth or out_tokens")
        max_depth = int(out_tokens.shape[1]) - 1
    D = int(max_depth)
    dev = target.device
    if out_tokens is None:
        out_tokens = torch.empty((B, D + 1), dtype=torch.int32, device=dev)
    if out_accept_len is None:
        out_accept_len = torch.empty((B,), dtype=torch.int32, device=dev)
    if tuple(out_tokens.shape) != (B, D + 1) or tuple(out_accept_len.shape) != (B,):
        raise ValueError("output shapes do not match [B, D+1] / [B]")
    if seq_stride is None and target.numel() != B * (N + 1) * V:
        raise ValueError("target must be [B, N+1, V] (or pass seq_stride)")
    o = make_opts(mode, cluster_size, block_threads, no_tma, seq_stride, status, out_nodes,
                  out_dist, out_rejects, prefetch, kernel, z_rule, proxy_denominator, fill)
    o.parents_stride = N if per_seq_tree else 0
    if out_phase is not None:
        _need_cuda("out_phase", out_phase)
        if out_phase.dtype != torch.int64 or tuple(out_phase.shape) != (B, len(PHASES)):
            raise ValueError("out_phase must be int64 [B, 6]")
        o.out_phase_cycles = out_phase.data_ptr()
    if out_candidates is not None:
        if out_candidates.dtype != torch.int32 or tuple(out_candidates.shape) != (B, N):
            raise ValueError("out_candidates must be int32 [B, N]")
        o.out_candidates = out_candidates.data_ptr()
    if stream is None:
        stream = torch.cuda.current_stream(dev)
    handle = stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)
    d = Dims(B, N, V, D, dt)
    rc = lib.resispec_verify_ex(_ptr(target), _ptr(draft), _ptr(tree_parents),
                                _ptr(cand_tokens), ctypes.c_float(float(temperature)),
                                ctypes.c_uint64(int(seed) & 0xFFFFFFFFFFFFFFFF),
                                _ptr(out_tokens), _ptr(out_accept_len), d, ctypes.byref(o),
                                ctypes.c_void_p(handle))
    if rc:
        raise ResispecError(rc, "resispec_verify_ex")
    return out_tokens, out_accept_len


def uniforms(seed, seq, row, stream=None):
    """Device Philox draws U(seed, seq[i], row[i], 0 / 1) for tests."""
    torch = _torch()
    lib = load_library()
    _need_cuda("seq", seq)
    _need_cuda("row", row)
    n = int(seq.numel())
    u0 = torch.empty(n, dtype=torch.float32, device=seq.device)
    u1 = torch.empty(n, dtype=torch.float32, device=seq.device)
    if stream is None:
        stream = torch.cuda.current_stream(seq.device)
    rc = lib.resispec_uniforms(ctypes.c_uint64(int(seed) & 0xFFFFFFFFFFFFFFFF), _ptr(seq),
                               _ptr(row), n, _ptr(u0), _ptr(u1),
                               ctypes.c_void_p(stream.cuda_stream))
    if rc:
        raise ResispecError(rc, "resispec_uniforms")
    return u0, u1
