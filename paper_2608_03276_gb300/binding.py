"""ctypes binding of libtaskpress.so (include/taskpress.h), same names as the C ABI.

Argument marshalling only: every wrapper checks the torch tensors it is given
(device, dtype, contiguity, size), passes raw pointers and the current CUDA
stream, and raises on a non-zero status.  All arithmetic runs in the library's
kernels; there is no fallback when the library is missing.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_double, c_float, c_int, c_int32, c_int64, c_size_t, c_uint32, c_void_p
from typing import Optional, Sequence

import numpy as np

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libtaskpress.so")

TP_OK = 0
TP_ERR_INVALID_ARG = -1
TP_ERR_WORKSPACE = -2
TP_ERR_UNSUPPORTED_SHAPE = -3
TP_ERR_CUDA = -4
TP_ERR_TIMEOUT = -5
TP_SCORE_KEY_ONLY = 0x1
TP_SCORE_NORM_ADD = 0x2
TP_SCORE_HARMONIC = 0x4
TP_MAX_BATCH = 256
TP_MAX_ROWS = 512
TP_MAX_GUIDE_ROWS = 8192
#: every symbol include/taskpress.h declares
EXPORTS = ("tp_budget", "tp_kept_capacity", "tp_workspace_bytes", "tp_quantize_v",
           "tp_guide_scores", "tp_guide_lse", "tp_guide_lse_static", "tp_guide_key_scores",
           "tp_select", "tp_compact",
           "tp_compress_layer", "tp_compress_layer_lse", "tp_guide_prefix_lse",
           "tp_compress_layer_guide", "tp_compress_layers", "tp_quantize_rows", "tp_check_status",
           "tp_selftest_wait_timeout", "tp_status_string", "tp_compress_kernel_count",
           "tp_compress_layers_lse", "tp_workspace_bytes_stack", "tp_stack_layers_per_selection")


class TpProblem(ctypes.Structure):
    _fields_ = [
        ("n_heads_q", c_int32),
        ("n_heads_kv", c_int32),
        ("head_dim", c_int32),
        ("guide_len", c_int32),
        ("batch", c_int32),
        ("pool_kernel", c_int32),
        ("quant_bits", c_int32),
        ("softmax_scale", c_float),
        ("flags", c_uint32),
        ("doc_offsets", POINTER(c_int64)),
    ]


class TaskPressError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} failed: {status} ({_status_string(status)})")


_lib = None


def load(path: Optional[str] = None):
    """Loads libtaskpress.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"libtaskpress.so not built ({p}); run __graft_entry__.build()")
    lib = ctypes.CDLL(p)
    lib.tp_budget.restype = c_int64
    lib.tp_budget.argtypes = [c_int64, c_double]
    lib.tp_kept_capacity.restype = c_int64
    lib.tp_kept_capacity.argtypes = [POINTER(TpProblem), c_double, c_int64]
    lib.tp_workspace_bytes.restype = c_size_t
    lib.tp_workspace_bytes.argtypes = [POINTER(TpProblem), c_double, c_int64]
    lib.tp_workspace_bytes_stack.restype = c_size_t
    lib.tp_workspace_bytes_stack.argtypes = [POINTER(TpProblem), c_double, c_int64, c_int]
    lib.tp_stack_layers_per_selection.restype = c_int
    lib.tp_stack_layers_per_selection.argtypes = [POINTER(TpProblem), c_double, c_int64, c_int, c_size_t]
    lib.tp_quantize_v.restype = c_int
    lib.tp_quantize_v.argtypes = [POINTER(TpProblem), c_void_p, c_void_p, c_void_p, c_void_p]
    lib.tp_guide_scores.restype = c_int
    lib.tp_guide_scores.argtypes = [POINTER(TpProblem), c_void_p, c_void_p, c_void_p, c_void_p,
                                    c_void_p, c_size_t, c_void_p]
    lib.tp_guide_lse.restype = c_int
    lib.tp_guide_lse.argtypes = [POINTER(TpProblem), c_void_p, c_void_p, c_void_p, c_void_p,
                                 c_void_p, c_void_p, c_size_t, c_void_p]
    lib.tp_guide_lse_static.restype = c_int
    lib.tp_guide_lse_static.argtypes = [POINTER(TpProblem), c_void_p, c_void_p, c_void_p, c_void_p,
                                        c_void_p, c_void_p]
    lib.tp_guide_key_scores.restype = c_int
    lib.tp_guide_key_scores.argtypes = [POINTER(TpProblem), c_void_p, c_void_p, c_void_p, c_void_p,
                                        c_void_p, c_void_p, c_void_p]
    lib.tp_select.restype = c_int
    lib.tp_select.argtypes = [POINTER(TpProblem), c_void_p, c_double, c_int64, c_void_p, c_void_p,
                              c_size_t, c_void_p]
    lib.tp_compact.restype = c_int
    lib.tp_compact.argtypes = [POINTER(TpProblem), c_void_p, c_void_p, c_void_p, c_void_p, c_double,
                               c_int64, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]
    lib.tp_compress_layer.restype = c_int
    lib.tp_compress_layer.argtypes = [POINTER(TpProblem), c_void_p, c_void_p, c_void_p, c_double,
                                      c_int64, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                      c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]
    lib.tp_compress_layer_lse.restype = c_int
    lib.tp_compress_layer_lse.argtypes = [POINTER(TpProblem), c_void_p, c_void_p, c_void_p, c_void_p,
                                          c_double, c_int64, c_void_p, c_void_p, c_void_p, c_void_p,
                                          c_void_p, c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]
    lib.tp_guide_prefix_lse.restype = c_int
    lib.tp_guide_prefix_lse.argtypes = [POINTER(TpProblem), c_void_p, c_void_p, c_void_p, c_void_p]
    lib.tp_compress_layer_guide.restype = c_int
    lib.tp_compress_layer_guide.argtypes = lib.tp_compress_layer_lse.argtypes
    lib.tp_compress_layers.restype = c_int
    lib.tp_compress_layers.argtypes = [POINTER(TpProblem), c_int, c_void_p, c_void_p, c_void_p, c_double,
                                       c_int64, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                       c_void_p, c_size_t, c_void_p]
    lib.tp_quantize_rows.restype = c_int
    lib.tp_quantize_rows.argtypes = [c_void_p, c_int64, c_int, c_int, c_void_p, c_void_p, c_void_p]
    lib.tp_selftest_wait_timeout.restype = c_int
    lib.tp_selftest_wait_timeout.argtypes = [c_void_p, c_size_t, c_int64, c_void_p]
    lib.tp_check_status.restype = c_int
    lib.tp_check_status.argtypes = [c_void_p, c_size_t, c_void_p]
    lib.tp_status_string.restype = ctypes.c_char_p
    lib.tp_status_string.argtypes = [c_int]
    lib.tp_compress_layers_lse.restype = c_int
    lib.tp_compress_layers_lse.argtypes = [POINTER(TpProblem), c_int, c_void_p, c_void_p, c_void_p,
                                           c_void_p, c_double, c_int64, c_void_p, c_void_p, c_void_p,
                                           c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]
    lib.tp_compress_kernel_count.restype = c_int
    lib.tp_compress_kernel_count.argtypes = [POINTER(TpProblem), c_double, c_int64, c_int]
    _lib = lib
    return lib


def _status_string(status: int) -> str:
    try:
        return load().tp_status_string(status).decode()
    except Exception:
        return "?"


class Problem:
    """A tp_problem plus the host offsets array it points to (kept alive here)."""

    def __init__(self, n_heads_q: int, n_heads_kv: int, head_dim: int, guide_len: int,
                 doc_offsets: Sequence[int], pool_kernel: int = 5, quant_bits: int = 8,
                 softmax_scale: float = 0.0, flags: int = 0):
        self.offsets = np.ascontiguousarray(np.asarray(doc_offsets, dtype=np.int64))
        self.c = TpProblem(n_heads_q, n_heads_kv, head_dim, guide_len, len(self.offsets) - 1,
                           pool_kernel, quant_bits, softmax_scale, flags,
                           self.offsets.ctypes.data_as(POINTER(c_int64)))

    @property
    def n_total(self) -> int:
        return int(self.offsets[-1])

    @property
    def batch(self) -> int:
        return len(self.offsets) - 1

    def ref(self):
        return ctypes.byref(self.c)


def _ptr(t, dtype=None, numel=None, name="tensor", nullable=False):
    if t is None:
        if nullable:
            return None
        raise ValueError(f"{name} is required")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if numel is not None and t.numel() != numel:
        raise ValueError(f"{name} must have {numel} elements, got {t.numel()}")
    return c_void_p(t.data_ptr())


def _codes(p: Problem, t, rows: int, name: str):
    """Eq. 2 code buffer of `rows` rows: int8 [rows, d] at b = 8, uint8
    [rows, d / 2] (two codes per byte) at b = 4; None allowed."""
    import torch
    bits, d = p.c.quant_bits, p.c.head_dim
    return _ptr(t, torch.int8 if bits == 8 else torch.uint8, rows * d * bits // 8, name, nullable=True)


def code_dtype(p: Problem):
    import torch
    return torch.int8 if p.c.quant_bits == 8 else torch.uint8


def _stream(stream):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return c_void_p(s.cuda_stream)


def _check(fn: str, status: int):
    if status != TP_OK:
        raise TaskPressError(fn, status)


def tp_budget(n: int, keep_ratio: float) -> int:
    return int(load().tp_budget(n, keep_ratio))


def tp_kept_capacity(p: Problem, keep_ratio: float, budget: int) -> int:
    return int(load().tp_kept_capacity(p.ref(), keep_ratio, budget))


def tp_workspace_bytes(p: Problem, keep_ratio: float = 0.0, budget: int = 0) -> int:
    return int(load().tp_workspace_bytes(p.ref(), keep_ratio, budget))


def tp_workspace_bytes_stack(p: Problem, keep_ratio: float, budget: int, n_layers: int) -> int:
    return int(load().tp_workspace_bytes_stack(p.ref(), keep_ratio, budget, n_layers))


def tp_stack_layers_per_selection(p: Problem, keep_ratio: float, budget: int, n_layers: int,
                                  ws_bytes: int) -> int:
    n = int(load().tp_stack_layers_per_selection(p.ref(), keep_ratio, budget, n_layers, ws_bytes))
    if n < 0:
        raise TaskPressError("tp_stack_layers_per_selection", TP_ERR_INVALID_ARG)
    return n


def tp_quantize_v(p: Problem, v, vq, gamma, stream=None):
    import torch
    hkv, d, n = p.c.n_heads_kv, p.c.head_dim, p.n_total
    _check("tp_quantize_v", load().tp_quantize_v(
        p.ref(), _ptr(v, torch.bfloat16, hkv * n * d, "v"),
        _codes(p, vq, hkv * n, "vq"),
        _ptr(gamma, torch.float32, hkv * n, "gamma"), _stream(stream)))


def tp_quantize_rows(x, quant_bits: int, xq, scale, stream=None):
    """Eq. 2 for every row of `x` ([..., d] bf16): per-row scales `scale`
    ([...] fp32) and codes `xq` ([..., d*quant_bits/8], int8 at 8 bits, uint8
    two per byte at 4 bits; None to skip)."""
    import torch
    d = x.shape[-1]
    rows = x.numel() // d
    _check("tp_quantize_rows", load().tp_quantize_rows(
        _ptr(x, torch.bfloat16, None, "x"), rows, d, quant_bits,
        _ptr(xq, torch.int8 if quant_bits == 8 else torch.uint8, rows * d * quant_bits // 8, "xq",
             nullable=True),
        _ptr(scale, torch.float32, rows, "scale"), _stream(stream)))


def tp_guide_scores(p: Problem, q, k, gamma, scores, ws, stream=None):
    import torch
    hq, hkv, d, lt, n = p.c.n_heads_q, p.c.n_heads_kv, p.c.head_dim, p.c.guide_len, p.n_total
    _check("tp_guide_scores", load().tp_guide_scores(
        p.ref(), _ptr(q, torch.bfloat16, p.batch * hq * lt * d, "q"),
        _ptr(k, torch.bfloat16, hkv * n * d, "k"),
        _ptr(gamma, torch.float32, hkv * n, "gamma", nullable=True),
        _ptr(scores, torch.float32, hkv * n, "scores"),
        _ptr(ws, torch.uint8, None, "ws"), ws.numel(), _stream(stream)))


def tp_guide_lse(p: Problem, q, k, lse, ws, stream=None, v=None, gamma=None):
    import torch
    hq, hkv, d, lt, n = p.c.n_heads_q, p.c.n_heads_kv, p.c.head_dim, p.c.guide_len, p.n_total
    rows = (hq // hkv) * lt
    _check("tp_guide_lse", load().tp_guide_lse(
        p.ref(), _ptr(q, torch.bfloat16, p.batch * hq * lt * d, "q"),
        _ptr(k, torch.bfloat16, hkv * n * d, "k"),
        _ptr(v, torch.bfloat16, hkv * n * d, "v", nullable=True),
        _ptr(lse, torch.float32, p.batch * hkv * rows, "lse"),
        _ptr(gamma, torch.float32, hkv * n, "gamma", nullable=True),
        _ptr(ws, torch.uint8, None, "ws"), ws.numel(), _stream(stream)))


def tp_guide_lse_static(p: Problem, q, k, lse, stream=None, v=None, gamma=None):
    """tp_guide_lse with the library's fixed device scratch (no workspace argument)."""
    import torch
    hq, hkv, d, lt, n = p.c.n_heads_q, p.c.n_heads_kv, p.c.head_dim, p.c.guide_len, p.n_total
    rows = (hq // hkv) * lt
    _check("tp_guide_lse_static", load().tp_guide_lse_static(
        p.ref(), _ptr(q, torch.bfloat16, p.batch * hq * lt * d, "q"),
        _ptr(k, torch.bfloat16, hkv * n * d, "k"),
        _ptr(v, torch.bfloat16, hkv * n * d, "v", nullable=True),
        _ptr(lse, torch.float32, p.batch * hkv * rows, "lse"),
        _ptr(gamma, torch.float32, hkv * n, "gamma", nullable=True), _stream(stream)))


def tp_guide_key_scores(p: Problem, q, k, lse, key_scores, stream=None, v=None, gamma=None):
    import torch
    hq, hkv, d, lt, n = p.c.n_heads_q, p.c.n_heads_kv, p.c.head_dim, p.c.guide_len, p.n_total
    rows = (hq // hkv) * lt
    _check("tp_guide_key_scores", load().tp_guide_key_scores(
        p.ref(), _ptr(q, torch.bfloat16, p.batch * hq * lt * d, "q"),
        _ptr(k, torch.bfloat16, hkv * n * d, "k"),
        _ptr(v, torch.bfloat16, hkv * n * d, "v", nullable=True),
        _ptr(lse, torch.float32, p.batch * hkv * rows, "lse"),
        _ptr(key_scores, torch.float32, hkv * n, "key_scores"),
        _ptr(gamma, torch.float32, hkv * n, "gamma", nullable=True), _stream(stream)))


def tp_guide_prefix_lse(p: Problem, q, k_guide, lse, stream=None):
    """Folds the guide's causal prefix into the row normalisers `lse`, in place."""
    import torch
    hq, hkv, d, lt = p.c.n_heads_q, p.c.n_heads_kv, p.c.head_dim, p.c.guide_len
    rows = (hq // hkv) * lt
    _check("tp_guide_prefix_lse", load().tp_guide_prefix_lse(
        p.ref(), _ptr(q, torch.bfloat16, p.batch * hq * lt * d, "q"),
        _ptr(k_guide, torch.bfloat16, p.batch * hkv * lt * d, "k_guide"),
        _ptr(lse, torch.float32, p.batch * hkv * rows, "lse"), _stream(stream)))


def tp_select(p: Problem, scores, keep_ratio: float, budget: int, idx, ws, stream=None):
    import torch
    hkv, n = p.c.n_heads_kv, p.n_total
    cap = tp_kept_capacity(p, keep_ratio, budget)
    _check("tp_select", load().tp_select(
        p.ref(), _ptr(scores, torch.float32, hkv * n, "scores"), keep_ratio, budget,
        _ptr(idx, torch.int32, p.batch * hkv * cap, "idx", nullable=cap == 0),
        _ptr(ws, torch.uint8, None, "ws"), ws.numel(), _stream(stream)))


def tp_compact(p: Problem, k, v, gamma, idx, keep_ratio: float, budget: int, kc, vc, vqc, gammac,
               stream=None):
    import torch
    hkv, d, n = p.c.n_heads_kv, p.c.head_dim, p.n_total
    cap = tp_kept_capacity(p, keep_ratio, budget)
    m = p.batch * hkv * cap
    _check("tp_compact", load().tp_compact(
        p.ref(), _ptr(k, torch.bfloat16, hkv * n * d, "k"), _ptr(v, torch.bfloat16, hkv * n * d, "v"),
        _ptr(gamma, torch.float32, hkv * n, "gamma"), _ptr(idx, torch.int32, m, "idx"),
        keep_ratio, budget,
        _ptr(kc, torch.bfloat16, m * d, "kc", nullable=True),
        _ptr(vc, torch.bfloat16, m * d, "vc", nullable=True),
        _codes(p, vqc, m, "vqc"),
        _ptr(gammac, torch.float32, m, "gammac", nullable=True), _stream(stream)))


def tp_compress_layer(p: Problem, q, k, v, keep_ratio: float, budget: int, idx, kc, vc, vqc, gammac,
                      scores, gamma, ws, stream=None):
    import torch
    hq, hkv, d, lt, n = p.c.n_heads_q, p.c.n_heads_kv, p.c.head_dim, p.c.guide_len, p.n_total
    cap = tp_kept_capacity(p, keep_ratio, budget)
    m = p.batch * hkv * cap
    _check("tp_compress_layer", load().tp_compress_layer(
        p.ref(), _ptr(q, torch.bfloat16, p.batch * hq * lt * d, "q"),
        _ptr(k, torch.bfloat16, hkv * n * d, "k"), _ptr(v, torch.bfloat16, hkv * n * d, "v"),
        keep_ratio, budget,
        _ptr(idx, torch.int32, m, "idx", nullable=cap == 0),
        _ptr(kc, torch.bfloat16, m * d, "kc", nullable=True),
        _ptr(vc, torch.bfloat16, m * d, "vc", nullable=True),
        _codes(p, vqc, m, "vqc"),
        _ptr(gammac, torch.float32, m, "gammac", nullable=True),
        _ptr(scores, torch.float32, hkv * n, "scores", nullable=True),
        _ptr(gamma, torch.float32, hkv * n, "gamma", nullable=True),
        _ptr(ws, torch.uint8, None, "ws"), ws.numel(), _stream(stream)))


def tp_compress_layer_lse(p: Problem, q, k, v, lse, keep_ratio: float, budget: int, idx, kc, vc, vqc,
                          gammac, scores, gamma, ws, stream=None):
    import torch
    hq, hkv, d, lt, n = p.c.n_heads_q, p.c.n_heads_kv, p.c.head_dim, p.c.guide_len, p.n_total
    rows = (hq // hkv) * lt
    cap = tp_kept_capacity(p, keep_ratio, budget)
    m = p.batch * hkv * cap
    _check("tp_compress_layer_lse", load().tp_compress_layer_lse(
        p.ref(), _ptr(q, torch.bfloat16, p.batch * hq * lt * d, "q"),
        _ptr(k, torch.bfloat16, hkv * n * d, "k"), _ptr(v, torch.bfloat16, hkv * n * d, "v"),
        _ptr(lse, torch.float32, p.batch * hkv * rows, "lse"),
        keep_ratio, budget,
        _ptr(idx, torch.int32, m, "idx", nullable=cap == 0),
        _ptr(kc, torch.bfloat16, m * d, "kc", nullable=True),
        _ptr(vc, torch.bfloat16, m * d, "vc", nullable=True),
        _codes(p, vqc, m, "vqc"),
        _ptr(gammac, torch.float32, m, "gammac", nullable=True),
        _ptr(scores, torch.float32, hkv * n, "scores", nullable=True),
        _ptr(gamma, torch.float32, hkv * n, "gamma", nullable=True),
        _ptr(ws, torch.uint8, None, "ws"), ws.numel(), _stream(stream)))


def tp_compress_layer_guide(p: Problem, q, k, v, k_guide, keep_ratio: float, budget: int, idx, kc,
                            vc, vqc, gammac, scores, gamma, ws, stream=None):
    import torch
    hq, hkv, d, lt, n = p.c.n_heads_q, p.c.n_heads_kv, p.c.head_dim, p.c.guide_len, p.n_total
    cap = tp_kept_capacity(p, keep_ratio, budget)
    m = p.batch * hkv * cap
    _check("tp_compress_layer_guide", load().tp_compress_layer_guide(
        p.ref(), _ptr(q, torch.bfloat16, p.batch * hq * lt * d, "q"),
        _ptr(k, torch.bfloat16, hkv * n * d, "k"), _ptr(v, torch.bfloat16, hkv * n * d, "v"),
        _ptr(k_guide, torch.bfloat16, p.batch * hkv * lt * d, "k_guide"),
        keep_ratio, budget,
        _ptr(idx, torch.int32, m, "idx", nullable=cap == 0),
        _ptr(kc, torch.bfloat16, m * d, "kc", nullable=True),
        _ptr(vc, torch.bfloat16, m * d, "vc", nullable=True),
        _codes(p, vqc, m, "vqc"),
        _ptr(gammac, torch.float32, m, "gammac", nullable=True),
        _ptr(scores, torch.float32, hkv * n, "scores", nullable=True),
        _ptr(gamma, torch.float32, hkv * n, "gamma", nullable=True),
        _ptr(ws, torch.uint8, None, "ws"), ws.numel(), _stream(stream)))


def tp_compress_layers(p: Problem, layers, keep_ratio: float, budget: int, outs, ws, stream=None):
    """A stack of layers in one call.  `layers`: a sequence of (q, k, v) device
    tensors; `outs`: one CompressOutputs per layer (its idx, kc, vc, vqc and
    gammac are written; scores and gamma are not)."""
    import torch
    n = len(layers)
    if len(outs) != n:
        raise ValueError("one CompressOutputs per layer")
    hq, hkv, d, lt, nt = p.c.n_heads_q, p.c.n_heads_kv, p.c.head_dim, p.c.guide_len, p.n_total
    cap = tp_kept_capacity(p, keep_ratio, budget)
    m = p.batch * hkv * cap

    def arr(ptrs):
        a = (c_void_p * max(1, n))()
        for i, x in enumerate(ptrs):
            a[i] = x
        return a

    q = arr(_ptr(x[0], torch.bfloat16, p.batch * hq * lt * d, "q") for x in layers)
    k = arr(_ptr(x[1], torch.bfloat16, hkv * nt * d, "k") for x in layers)
    v = arr(_ptr(x[2], torch.bfloat16, hkv * nt * d, "v") for x in layers)
    idx = arr(_ptr(o.idx, torch.int32, m, "idx", nullable=cap == 0) for o in outs)
    kc = arr(_ptr(o.kc, torch.bfloat16, m * d, "kc", nullable=True) for o in outs)
    vc = arr(_ptr(o.vc, torch.bfloat16, m * d, "vc", nullable=True) for o in outs)
    vqc = arr(_codes(p, o.vqc, m, "vqc") for o in outs)
    gc = arr(_ptr(o.gammac, torch.float32, m, "gammac", nullable=True) for o in outs)
    _check("tp_compress_layers", load().tp_compress_layers(
        p.ref(), n, q, k, v, keep_ratio, budget, idx, kc, vc, vqc, gc,
        _ptr(ws, torch.uint8, None, "ws"), ws.numel(), _stream(stream)))


def tp_compress_layers_lse(p: Problem, layers, lses, keep_ratio: float, budget: int, outs, ws,
                           stream=None):
    """A stack of layers with the caller's row normalisers: `lses` holds one
    [batch, H_kv, M] fp32 tensor per layer; otherwise as tp_compress_layers."""
    import torch
    n = len(layers)
    if len(outs) != n or len(lses) != n:
        raise ValueError("one CompressOutputs and one lse tensor per layer")
    hq, hkv, d, lt, nt = p.c.n_heads_q, p.c.n_heads_kv, p.c.head_dim, p.c.guide_len, p.n_total
    rows = (hq // hkv) * lt
    cap = tp_kept_capacity(p, keep_ratio, budget)
    m = p.batch * hkv * cap

    def arr(ptrs):
        a = (c_void_p * max(1, n))()
        for i, x in enumerate(ptrs):
            a[i] = x
        return a

    q = arr(_ptr(x[0], torch.bfloat16, p.batch * hq * lt * d, "q") for x in layers)
    k = arr(_ptr(x[1], torch.bfloat16, hkv * nt * d, "k") for x in layers)
    v = arr(_ptr(x[2], torch.bfloat16, hkv * nt * d, "v") for x in layers)
    ls = arr(_ptr(t, torch.float32, p.batch * hkv * rows, "lse") for t in lses)
    idx = arr(_ptr(o.idx, torch.int32, m, "idx", nullable=cap == 0) for o in outs)
    kc = arr(_ptr(o.kc, torch.bfloat16, m * d, "kc", nullable=True) for o in outs)
    vc = arr(_ptr(o.vc, torch.bfloat16, m * d, "vc", nullable=True) for o in outs)
    vqc = arr(_codes(p, o.vqc, m, "vqc") for o in outs)
    gc = arr(_ptr(o.gammac, torch.float32, m, "gammac", nullable=True) for o in outs)
    _check("tp_compress_layers_lse", load().tp_compress_layers_lse(
        p.ref(), n, q, k, v, ls, keep_ratio, budget, idx, kc, vc, vqc, gc,
        _ptr(ws, torch.uint8, None, "ws"), ws.numel(), _stream(stream)))


def tp_selftest_wait_timeout(ws, limit_ns: int, stream=None):
    """Runs the bounded-wait self-test: the status word of `ws` then reads
    TP_ERR_TIMEOUT (see tp_check_status)."""
    import torch
    _check("tp_selftest_wait_timeout", load().tp_selftest_wait_timeout(
        _ptr(ws, torch.uint8, None, "ws"), ws.numel(), int(limit_ns), _stream(stream)))


def tp_check_status(ws, stream=None) -> int:
    return int(load().tp_check_status(c_void_p(ws.data_ptr()), ws.numel(), _stream(stream)))


def tp_status_string(status: int) -> str:
    return _status_string(status)


#: tp_compress_kernel_count modes
MODE_TWO_PASS, MODE_CALLER_LSE, MODE_LITERAL = 0, 1, 2


def tp_compress_kernel_count(p: Problem, keep_ratio: float, budget: int, mode: int = MODE_TWO_PASS) -> int:
    """Kernels one fused call launches for this problem (a planning query)."""
    n = int(load().tp_compress_kernel_count(p.ref(), keep_ratio, budget, mode))
    if n < 0:
        raise TaskPressError("tp_compress_kernel_count", TP_ERR_INVALID_ARG)
    return n


class CompressOutputs:
    """Device buffers for one tp_compress_layer call (plumbing: torch allocations)."""

    def __init__(self, p: Problem, keep_ratio: float, budget: int, device, with_scores=True):
        import torch
        hkv, d, n = p.c.n_heads_kv, p.c.head_dim, p.n_total
        self.cap = tp_kept_capacity(p, keep_ratio, budget)
        if self.cap < 0:
            raise ValueError("invalid keep ratio / budget")
        shp = (p.batch, hkv, self.cap)
        self.idx = torch.empty(shp, dtype=torch.int32, device=device)
        self.kc = torch.empty(shp + (d,), dtype=torch.bfloat16, device=device)
        self.vc = torch.empty(shp + (d,), dtype=torch.bfloat16, device=device)
        self.vqc = torch.empty(shp + (d * p.c.quant_bits // 8,), dtype=code_dtype(p), device=device)
        self.gammac = torch.empty(shp, dtype=torch.float32, device=device)
        self.scores = torch.empty((hkv, n), dtype=torch.float32, device=device) if with_scores else None
        self.gamma = torch.empty((hkv, n), dtype=torch.float32, device=device) if with_scores else None
        self.ws = torch.empty(max(256, tp_workspace_bytes(p, keep_ratio, budget)), dtype=torch.uint8,
                              device=device)


def compress(p: Problem, q, k, v, keep_ratio: float, budget: int, out: CompressOutputs, stream=None,
             lse=None, k_guide=None):
    """One layer through tp_compress_layer; through tp_compress_layer_lse with
    the caller's row normalisers `lse`; or through tp_compress_layer_guide with
    the guide's keys `k_guide` (the literal normaliser)."""
    if lse is not None and k_guide is not None:
        raise ValueError("give either lse or k_guide")
    if k_guide is not None:
        tp_compress_layer_guide(p, q, k, v, k_guide, keep_ratio, budget, out.idx, out.kc, out.vc,
                                out.vqc, out.gammac, out.scores, out.gamma, out.ws, stream)
    elif lse is None:
        tp_compress_layer(p, q, k, v, keep_ratio, budget, out.idx, out.kc, out.vc, out.vqc,
                          out.gammac, out.scores, out.gamma, out.ws, stream)
    else:
        tp_compress_layer_lse(p, q, k, v, lse, keep_ratio, budget, out.idx, out.kc, out.vc, out.vqc,
                              out.gammac, out.scores, out.gamma, out.ws, stream)
    return out
