"""Python binding of librealq.so, the GB300 (sm_103a) REAL-Q per-layer sweep.

Every function here marshals torch tensors (device memory, current stream)
into the C ABI declared in include/realq.h and calls it; all computation runs
in the library's CUDA kernels.  There is no CPU fallback: if the library is
missing, importing the binding works but every call raises.

Names match the C entry points.  Errors come back as RealqError carrying the
status code and the library's message.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

__all__ = [
    "RealqError", "QuantCfg", "BgdCfg", "lib", "library_path", "quant_cfg", "bgd_cfg", "workspace",
    "realq_hessian_accumulate", "realq_hessian_workspace_size", "realq_hessian_prepare",
    "realq_prepare_workspace_size", "realq_hessian_prepare_noalloc",
    "realq_hessian_prepare_deferred", "realq_prepare_status", "Graph", "realq_graph_begin", "realq_graph_end", "realq_scale_moment", "realq_quantize_layer",
    "realq_quantize_activations", "realq_saliency_clip", "realq_hessian_weighted_workspace_size",
    "realq_hessian_accumulate_weighted", "realq_hessian_prepare_scaled", "realq_quantize_layer_grouped",
    "realq_quantize_grouped_workspace_size", "realq_quantize_layer_minibatch",
    "realq_quantize_minibatch_workspace_size", "realq_quantize_tokens_workspace_size", "realq_quantize_layer_tokens",
    "realq_quantize_trace_workspace_size",
    "realq_quantize_workspace_size", "realq_bgd_refine", "realq_bgd_workspace_size",
    "realq_surrogate_loss", "realq_surrogate_workspace_size", "realq_workspace_status",
    "realq_status_string", "realq_last_error", "realq_launch_count", "realq_profile_enable",
    "realq_profile_collect", "realq_reverse_cosine_lr", "realq_set_tensor_tile", "realq_set_quant_kernel", "realq_set_block_products", "realq_set_bgd_products", "realq_set_tensor_overlap", "realq_set_block_attention", "BlockDims", "block_dims", "realq_block_workspace_size", "realq_block_forward",
    "realq_block_window", "BLOCK_MODULES", "realq_block_module_workspace_size", "realq_block_head_workspace_size",
    "realq_block_module_window", "realq_block_head_kl", "realq_block_module_kl",
    "realq_quantize_window_workspace_size", "realq_quantize_layer_window", "realq_block_module_inputs",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
library_path = os.path.join(_HERE, "_lib", "librealq.so")

REALQ_OK, REALQ_ERR_INVALID_ARG, REALQ_ERR_WORKSPACE, REALQ_ERR_NOT_SPD = 0, 1, 2, 3
REALQ_ERR_NONFINITE, REALQ_ERR_TIMEOUT, REALQ_ERR_CUDA, REALQ_ERR_UNSUPPORTED = 4, 5, 6, 7
REALQ_F32, REALQ_BF16 = 0, 1
REALQ_OPT_ADAM, REALQ_OPT_SGD = 0, 1


class RealqError(RuntimeError):
    def __init__(self, status: int, message: str, **extra):
        super().__init__(f"realq status {status}: {message}")
        self.status = status
        self.message = message
        for k, v in extra.items():
            setattr(self, k, v)


class QuantCfg(ctypes.Structure):
    _fields_ = [("bits", ctypes.c_int), ("group_size", ctypes.c_int), ("block_size", ctypes.c_int),
                ("symmetric", ctypes.c_int), ("damp_frac", ctypes.c_float)]


class BgdCfg(ctypes.Structure):
    _fields_ = [("steps_per_block", ctypes.c_int), ("optimizer", ctypes.c_int), ("lr", ctypes.c_float),
                ("beta1", ctypes.c_float), ("beta2", ctypes.c_float), ("eps", ctypes.c_float),
                ("b_global_start", ctypes.c_int), ("B_total", ctypes.c_int)]


class BlockDims(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int64), ("n_heads", ctypes.c_int64), ("n_kv", ctypes.c_int64),
                ("head_dim", ctypes.c_int64), ("ffn", ctypes.c_int64), ("rms_eps", ctypes.c_float),
                ("rope_base", ctypes.c_float)]


class BlockWeights(ctypes.Structure):
    _fields_ = [(k, ctypes.c_void_p) for k in ("g1", "Wq", "Wk", "Wv", "Wo", "g2", "Wg", "Wu", "Wd")]


class KernelStat(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 48), ("launches", ctypes.c_int64), ("total_ms", ctypes.c_double)]


def quant_cfg(bits=4, group_size=128, block_size=128, symmetric=0, damp_frac=0.01) -> QuantCfg:
    return QuantCfg(bits, group_size, block_size, int(symmetric), damp_frac)


def bgd_cfg(lr, steps_per_block=1, optimizer=REALQ_OPT_ADAM, beta1=0.9, beta2=0.999, eps=1e-8,
            b_global_start=1, B_total=1) -> BgdCfg:
    return BgdCfg(steps_per_block, optimizer, lr, beta1, beta2, eps, b_global_start, B_total)


_lib = None
_vp, _i64, _sz, _int, _f32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_size_t, ctypes.c_int, ctypes.c_float
_f64 = ctypes.c_double
_P_i64 = ctypes.POINTER(ctypes.c_int64)
_SIGS = {
    "realq_hessian_accumulate": ([_vp, _i64, _i64, _vp, _vp, _int, _vp, _vp, _vp, _sz], _int),
    "realq_hessian_workspace_size": ([_i64, _i64, _int, _int], _sz),
    "realq_hessian_prepare": ([_vp, _i64, _i64, _f32, _vp, _vp, _vp, _vp, _P_i64, _vp, _sz], _int),
    "realq_prepare_workspace_size": ([_i64], _sz),
    "realq_hessian_prepare_noalloc": ([_vp, _i64, _i64, _f32, _vp, _vp, _vp, _vp, _P_i64], _int),
    "realq_hessian_prepare_deferred": ([_vp, _i64, _i64, _f32, _vp, _vp, _vp, _vp, _vp, _sz], _int),
    "realq_prepare_status": ([_vp, _vp, _sz, _P_i64], _int),
    "realq_graph_begin": ([_vp], _int),
    "realq_graph_end": ([_vp, _int, ctypes.POINTER(_vp)], _int),
    "realq_graph_launch": ([_vp, _vp], _int),
    "realq_graph_kernels": ([_vp], _i64),
    "realq_graph_destroy": ([_vp], None),
    "realq_scale_moment": ([_vp, _i64, _i64, _vp, _vp], _int),
    "realq_quantize_activations": ([_vp, _i64, _i64, _vp, _int, _int, _f32, _vp, _vp, _vp], _int),
    "realq_saliency_clip": ([_vp, _i64, _int, _vp, _f64, _vp, _vp], _int),
    "realq_hessian_weighted_workspace_size": ([_i64, _i64], _sz),
    "realq_hessian_accumulate_weighted": ([_vp, _i64, _i64, _vp, _int, _vp, _vp, _vp, _vp, _sz], _int),
    "realq_hessian_prepare_scaled": ([_vp, _i64, ctypes.c_double, _f32, _vp, _vp, _vp, _vp, _P_i64, _vp, _sz], _int),
    "realq_quantize_grouped_workspace_size": ([_i64, _i64, _int, ctypes.POINTER(QuantCfg), ctypes.POINTER(BgdCfg),
                                               _int, _int], _sz),
    "realq_quantize_layer_grouped": ([_vp, _i64, _i64, _vp, _int, _int, _vp, _vp, _vp, _vp, _vp,
                                      ctypes.POINTER(QuantCfg), ctypes.POINTER(BgdCfg), _vp, _vp, _vp, _vp, _vp, _vp,
                                      _P_i64, _vp, _vp, _vp, _vp, _int, _i64, _i64, _vp, _sz], _int),
    "realq_quantize_minibatch_workspace_size": ([_i64, _i64, _int, ctypes.POINTER(QuantCfg), ctypes.POINTER(BgdCfg),
                                                 _int], _sz),
    "realq_quantize_layer_traced": ([_vp, _i64, _i64, _vp, _int, _vp, _vp, _vp, ctypes.POINTER(QuantCfg),
                                     ctypes.POINTER(BgdCfg), _vp, _vp, _vp, _vp, _vp, _vp, _P_i64, _vp, _vp, _vp, _vp,
                                     _int, _i64, _i64, _vp, _sz, _vp, _vp, _sz], _int),
    "realq_quantize_trace_workspace_size": ([_i64, _i64], _sz),
    "realq_quantize_tokens_workspace_size": ([_i64, _i64, _i64, ctypes.POINTER(QuantCfg), ctypes.POINTER(BgdCfg),
                                              _int], _sz),
    "realq_quantize_layer_tokens": ([_vp, _i64, _i64, _vp, _int, _vp, _vp, _vp, _vp, _i64, _i64, _f64,
                                     ctypes.POINTER(QuantCfg), ctypes.POINTER(BgdCfg), _vp, _vp, _vp, _vp, _vp, _vp,
                                     _P_i64, _vp, _vp, _vp, _vp, _int, _i64, _i64, _vp, _sz], _int),
    "realq_quantize_layer_minibatch": ([_vp, _i64, _i64, _vp, _int, _vp, _vp, _vp, _int, _vp,
                                        ctypes.POINTER(QuantCfg), ctypes.POINTER(BgdCfg), _vp, _vp, _vp, _vp, _vp,
                                        _vp, _P_i64, _vp, _vp, _vp, _vp, _int, _i64, _i64, _vp, _sz], _int),
    "realq_quantize_layer": ([_vp, _i64, _i64, _vp, _int, _vp, _vp, _vp, _vp, ctypes.POINTER(QuantCfg),
                              ctypes.POINTER(BgdCfg), _vp, _vp, _vp, _vp, _vp, _vp, _P_i64, _vp, _vp, _vp, _vp, _int,
                              _i64, _i64, _vp, _sz], _int),
    "realq_quantize_workspace_size": ([_i64, _i64, ctypes.POINTER(QuantCfg), ctypes.POINTER(BgdCfg), _int, _int],
                                      _sz),
    "realq_bgd_refine": ([_vp, _i64, _i64, _i64, _vp, _vp, _int, _vp, _vp, _vp, _vp, _f32, _vp, _vp, _P_i64,
                          ctypes.POINTER(BgdCfg), _vp, _sz], _int),
    "realq_bgd_workspace_size": ([_i64, _i64, _int, _int], _sz),
    "realq_surrogate_loss": ([_vp, _i64, _i64, _vp, _vp, _int, _vp, _vp, _vp, _vp, _sz], _int),
    "realq_surrogate_workspace_size": ([_i64, _i64], _sz),
    "realq_workspace_status": ([_vp, _vp, _sz], _int),
    "realq_block_workspace_size": ([ctypes.POINTER(BlockDims), _i64, _i64], _sz),
    "realq_set_tensor_tile": ([_int], _int),
    "realq_set_quant_kernel": ([_int], _int),
    "realq_set_block_products": ([_int], _int),
    "realq_set_bgd_products": ([_int], _int),
    "realq_set_tensor_overlap": ([_int], _int),
    "realq_set_block_attention": ([_int], _int),
    "realq_reverse_cosine_lr": ([_i64, _i64, _f64, ctypes.POINTER(ctypes.c_double)], _int),
    "realq_block_forward": ([_vp, ctypes.POINTER(BlockDims), ctypes.POINTER(BlockWeights), _i64, _i64, _vp, _vp,
                             _vp, _sz], _int),
    "realq_block_window": ([_vp, ctypes.POINTER(BlockDims), ctypes.POINTER(BlockWeights), _i64, _i64, _vp, _vp, _vp,
                            _vp, _vp, _vp, _sz], _int),
    "realq_block_module_workspace_size": ([ctypes.POINTER(BlockDims), _i64, _i64, _i64], _sz),
    "realq_block_head_workspace_size": ([_i64, _i64, _i64, _i64], _sz),
    "realq_block_module_window": ([_vp, ctypes.POINTER(BlockDims), ctypes.POINTER(BlockWeights),
                                   ctypes.POINTER(BlockWeights), ctypes.POINTER(BlockWeights), _i64, _i64, _vp, _vp,
                                   _int, _vp, _f32, _vp, _vp, _vp, _vp, _vp, _sz], _int),
    "realq_block_head_kl": ([_vp, _i64, _i64, _i64, _vp, _vp, _i64, _f32, _vp, _vp, _vp, _vp, _vp, _sz], _int),
    "realq_block_module_kl": ([_vp, ctypes.POINTER(BlockDims), ctypes.POINTER(BlockWeights),
                               ctypes.POINTER(BlockWeights), _i64, _i64, _vp, _vp, _int, _vp, _vp, _vp, _i64, _vp, _vp,
                               _vp, _sz], _int),
    "realq_block_module_inputs": ([_vp, ctypes.POINTER(BlockDims), ctypes.POINTER(BlockWeights), _i64, _i64, _vp,
                                   _int, _vp, _vp, _sz], _int),
    "realq_quantize_window_workspace_size": ([ctypes.POINTER(BlockDims), _i64, _i64, _int, _i64,
                                              ctypes.POINTER(QuantCfg)], _sz),
    "realq_quantize_layer_window": ([_vp, ctypes.POINTER(BlockDims), ctypes.POINTER(BlockWeights),
                                     ctypes.POINTER(BlockWeights), ctypes.POINTER(BlockWeights), _i64, _i64, _i64,
                                     _vp, _vp,
                                     _int, _vp, _vp, _vp, _vp, _i64,
                                     _vp, _vp, ctypes.POINTER(QuantCfg), ctypes.POINTER(BgdCfg), _vp, _vp, _vp, _P_i64,
                                     _vp, _vp, _vp, _vp, _int, _vp, _i64, _i64, _vp, _sz], _int),
    "realq_status_string": ([_int], ctypes.c_char_p),
    "realq_last_error": ([], ctypes.c_char_p),
    "realq_launch_count": ([], _i64),
    "realq_profile_enable": ([_int], None),
    "realq_profile_collect": ([ctypes.POINTER(KernelStat), _int], _int),
}


def lib():
    """The loaded CUDA library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(library_path):
            raise RuntimeError(f"{library_path} is missing: build it with paper_2609_00049_gb300.build.build() "
                               "(the CUDA library is required; there is no CPU fallback)")
        L = ctypes.CDLL(library_path)
        for name, (args, res) in _SIGS.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        _lib = L
    return _lib


def _check(status: int, **extra):
    if status != REALQ_OK:
        raise RealqError(status, lib().realq_last_error().decode(errors="replace"), **extra)


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return ctypes.c_void_p(t.data_ptr())


def _dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return REALQ_F32
    if t.dtype == torch.bfloat16:
        return REALQ_BF16
    raise ValueError(f"unsupported dtype {t.dtype}")


def _stream(stream) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _need(t, dtype, shape, name):
    if t is None:
        return
    if t.dtype != dtype or tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: expected {dtype} {tuple(shape)}, got {t.dtype} {tuple(t.shape)}")


def workspace(nbytes: int, device=None) -> Optional[torch.Tensor]:
    """Caller-owned workspace buffer (torch allocations are >= 256-byte aligned).
    Zeroed: its first word is the status that the kernels accumulate into and
    realq_workspace_status reads and clears."""
    if nbytes == 0:
        return None
    return torch.zeros(int(nbytes), dtype=torch.uint8, device=device or "cuda")


def _ws(ws):
    return (None, 0) if ws is None else (_ptr(ws), ws.numel())


# ----------------------------------------------------------------- Hessian ---
def realq_hessian_workspace_size(n: int, T_chunk: int, x_dtype: int = REALQ_BF16, has_X_fp: bool = False) -> int:
    return int(lib().realq_hessian_workspace_size(n, T_chunk, x_dtype, int(has_X_fp)))


def realq_hessian_accumulate(X_hat: torch.Tensor, H_sum: torch.Tensor, D_sum: Optional[torch.Tensor] = None,
                             X_fp: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None, stream=None):
    T, n = X_hat.shape
    _need(H_sum, torch.float32, (n, n), "H_sum")
    _need(D_sum, torch.float32, (n, n), "D_sum")
    if X_fp is not None and (X_fp.dtype != X_hat.dtype or X_fp.shape != X_hat.shape):
        raise ValueError("X_fp must match X_hat")
    wp, wb = _ws(ws)
    _check(lib().realq_hessian_accumulate(_stream(stream), n, T, _ptr(X_hat), _ptr(X_fp), _dtype(X_hat),
                                          _ptr(H_sum), _ptr(D_sum), wp, wb))


# ----------------------------------------------------------------- prepare ---
def realq_prepare_workspace_size(n: int) -> int:
    return int(lib().realq_prepare_workspace_size(n))


def realq_hessian_prepare(H_sum: torch.Tensor, T_total: int, damp_frac: float, U_out: torch.Tensor,
                          Hbar_out: Optional[torch.Tensor], dead_out: torch.Tensor, ws: torch.Tensor,
                          stream=None) -> int:
    """Returns -1; raises RealqError(status=NOT_SPD, fail_col=j) on a failed pivot."""
    n = H_sum.shape[0]
    _need(U_out, torch.float32, (n, n), "U_out")
    _need(Hbar_out, torch.float32, (n, n), "Hbar_out")
    _need(dead_out, torch.uint8, (n,), "dead_out")
    fc = ctypes.c_int64(-1)
    wp, wb = _ws(ws)
    st = lib().realq_hessian_prepare(_stream(stream), n, int(T_total), float(damp_frac), _ptr(H_sum), _ptr(U_out),
                                     _ptr(Hbar_out), _ptr(dead_out), ctypes.byref(fc), wp, wb)
    _check(st, fail_col=fc.value)
    return fc.value


def realq_hessian_prepare_deferred(H_sum: torch.Tensor, T_total: int, damp_frac: float, U_out: torch.Tensor,
                                   Hbar_out: Optional[torch.Tensor], dead_out: torch.Tensor, ws: torch.Tensor,
                                   stream=None) -> None:
    """realq_hessian_prepare that only enqueues (capturable into a CUDA graph);
    the factorisation status stays in ws, read with realq_prepare_status."""
    n = H_sum.shape[0]
    _need(U_out, torch.float32, (n, n), "U_out")
    _need(Hbar_out, torch.float32, (n, n), "Hbar_out")
    _need(dead_out, torch.uint8, (n,), "dead_out")
    wp, wb = _ws(ws)
    _check(lib().realq_hessian_prepare_deferred(_stream(stream), n, int(T_total), float(damp_frac), _ptr(H_sum),
                                                _ptr(U_out), _ptr(Hbar_out), _ptr(dead_out), wp, wb))


def realq_prepare_status(ws: torch.Tensor, stream=None) -> int:
    """Synchronizes; returns -1, or raises RealqError(status=NOT_SPD, fail_col=j)
    for the last prepare call on ws."""
    fc = ctypes.c_int64(-1)
    wp, wb = _ws(ws)
    st = lib().realq_prepare_status(_stream(stream), wp, wb, ctypes.byref(fc))
    _check(st, fail_col=fc.value)
    return fc.value


class Graph:
    """A captured step (realq_graph_t), destroyed with the object."""

    def __init__(self, handle: int):
        self.handle = handle

    @property
    def kernels(self) -> int:
        return int(lib().realq_graph_kernels(self.handle))

    def launch(self, stream=None) -> None:
        _check(lib().realq_graph_launch(self.handle, _stream(stream)))

    def __del__(self):
        if getattr(self, "handle", None) and _lib is not None:
            _lib.realq_graph_destroy(self.handle)
            self.handle = None


def realq_graph_begin(stream=None) -> None:
    """Start capturing `stream` (thread-local mode) into a graph."""
    _check(lib().realq_graph_begin(_stream(stream)))


def realq_graph_end(stream=None, node_priorities: bool = True) -> Graph:
    """End the capture of `stream`; with node_priorities the graph's kernels
    keep the priorities of the streams they were captured from."""
    h = ctypes.c_void_p()
    _check(lib().realq_graph_end(_stream(stream), int(bool(node_priorities)), ctypes.byref(h)))
    return Graph(h.value)


PREPARE_NOALLOC_MAX_N = 32768


def realq_hessian_prepare_noalloc(H_sum: torch.Tensor, T_total: int, damp_frac: float, U_out: torch.Tensor,
                                  Hbar_out: Optional[torch.Tensor], dead_out: torch.Tensor, stream=None) -> int:
    """realq_hessian_prepare without a workspace, for callers that cannot allocate
    device memory (its scratch is a fixed device array of the library, n <= 32768).
    Returns -1; raises RealqError(status=NOT_SPD, fail_col=j) on a failed pivot."""
    n = H_sum.shape[0]
    _need(U_out, torch.float32, (n, n), "U_out")
    _need(Hbar_out, torch.float32, (n, n), "Hbar_out")
    _need(dead_out, torch.uint8, (n,), "dead_out")
    fc = ctypes.c_int64(-1)
    st = lib().realq_hessian_prepare_noalloc(_stream(stream), n, int(T_total), float(damp_frac), _ptr(H_sum),
                                             _ptr(U_out), _ptr(Hbar_out), _ptr(dead_out), ctypes.byref(fc))
    _check(st, fail_col=fc.value)
    return fc.value


def realq_quantize_activations(X: torch.Tensor, bits: int = 4, a_clip: float = 0.9,
                               X_q: Optional[torch.Tensor] = None, codes: Optional[torch.Tensor] = None,
                               scale: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Per-token symmetric activation quantization (weight-activation setting).
    Returns X_q (allocated like X when not given; may be X itself)."""
    T, n = X.shape
    if X_q is None:
        X_q = torch.empty_like(X)
    _need(X_q, X.dtype, (T, n), "X_q")
    if codes is not None:
        _need(codes, torch.uint8, (T, (n + 1) // 2 if bits <= 4 else n), "codes")
    _need(scale, torch.float32, (T,), "scale")
    _check(lib().realq_quantize_activations(_stream(stream), T, n, _ptr(X), _dtype(X), bits, a_clip, _ptr(X_q),
                                            _ptr(codes), _ptr(scale)))
    return X_q


def realq_saliency_clip(S: torch.Tensor, pct: float = 0.99, S_out: Optional[torch.Tensor] = None,
                        clip_out: Optional[torch.Tensor] = None, stream=None):
    """Nearest-rank percentile of each saliency column and S clipped to it.
    Returns (S_out, clip_out); S_out may be S itself."""
    T, ng = S.shape
    _need(S, torch.float32, (T, ng), "S")
    if clip_out is None:
        clip_out = torch.empty(ng, dtype=torch.float32, device=S.device)
    if S_out is None:
        S_out = torch.empty_like(S)
    _need(S_out, torch.float32, (T, ng), "S_out")
    _check(lib().realq_saliency_clip(_stream(stream), T, ng, _ptr(S), pct, _ptr(S_out), _ptr(clip_out)))
    return S_out, clip_out


def realq_hessian_weighted_workspace_size(n: int, T_chunk: int) -> int:
    return int(lib().realq_hessian_weighted_workspace_size(n, T_chunk))


def realq_hessian_accumulate_weighted(X_hat: torch.Tensor, S: torch.Tensor, H_g: torch.Tensor, wsum: torch.Tensor,
                                      ws: torch.Tensor, stream=None):
    T, n = X_hat.shape
    ng = S.shape[1]
    if X_hat.dtype != torch.bfloat16:
        raise ValueError("X_hat: bf16 activations expected")
    _need(S, torch.float32, (T, ng), "S")
    _need(H_g, torch.float32, (ng, n, n), "H_g")
    _need(wsum, torch.float64, (ng,), "wsum")
    wp, wb = _ws(ws)
    _check(lib().realq_hessian_accumulate_weighted(_stream(stream), n, T, _ptr(X_hat), ng, _ptr(S), _ptr(H_g),
                                                   _ptr(wsum), wp, wb))


def realq_hessian_prepare_scaled(H_sum: torch.Tensor, norm: float, damp_frac: float, U_out: torch.Tensor,
                                 Hbar_out: Optional[torch.Tensor], dead_out: torch.Tensor, ws: torch.Tensor,
                                 stream=None) -> int:
    n = H_sum.shape[0]
    wp, wb = _ws(ws)
    fc = ctypes.c_int64(-1)
    _check(lib().realq_hessian_prepare_scaled(_stream(stream), n, float(norm), damp_frac, _ptr(H_sum), _ptr(U_out),
                                              _ptr(Hbar_out), _ptr(dead_out), ctypes.byref(fc), wp, wb),
           fail_col=fc.value)
    return fc.value


def realq_scale_moment(D_sum: torch.Tensor, T_total: int, Dbar: torch.Tensor, stream=None):
    n = D_sum.shape[0]
    _check(lib().realq_scale_moment(_stream(stream), n, int(T_total), _ptr(D_sum), _ptr(Dbar)))


# ------------------------------------------------------------------- sweep ---
def realq_quantize_workspace_size(m: int, n: int, qcfg: QuantCfg, bcfg: Optional[BgdCfg] = None,
                                  has_F_next: bool = False, has_Dbar: bool = False) -> int:
    return int(lib().realq_quantize_workspace_size(m, n, ctypes.byref(qcfg),
                                                   ctypes.byref(bcfg) if bcfg is not None else None,
                                                   int(has_F_next), int(has_Dbar)))


def realq_quantize_trace_workspace_size(m: int, n: int) -> int:
    return int(lib().realq_quantize_trace_workspace_size(m, n))


def realq_quantize_layer(W0: torch.Tensor, U: torch.Tensor, Hbar: Optional[torch.Tensor], qcfg: QuantCfg,
                         W_work: torch.Tensor, codes: torch.Tensor, scale: torch.Tensor, zero: torch.Tensor, *,
                         Dbar=None, dead=None, bcfg: Optional[BgdCfg] = None, F=None, F_next=None,
                         adam_m=None, adam_v=None, bgd_disp=None, adam_t: int = 0, W_deq=None,
                         block_begin: int = 0, block_end: Optional[int] = None, ws=None, stream=None,
                         block_loss: Optional[torch.Tensor] = None, trace_ws=None) -> int:
    """Runs blocks [block_begin, block_end) of the sweep; returns the Adam step counter.
    With block_loss (nb x 2 fp32, device) the surrogate before and after every
    block's Block-GD steps is written there (realq_quantize_layer_traced)."""
    m, n = W0.shape
    nb = -(-n // qcfg.block_size)
    if block_end is None:
        block_end = nb
    _need(W_work, torch.float32, (m, n), "W_work")
    _need(U, torch.float32, (n, n), "U")
    _need(codes, torch.uint8, (m, (n + 1) // 2), "codes")
    _need(adam_m, torch.float32, (m, n), "adam_m")
    _need(adam_v, torch.float32, (m, n), "adam_v")
    _need(bgd_disp, torch.float32, (m, n), "bgd_disp")
    t = ctypes.c_int64(adam_t)
    wp, wb = _ws(ws)
    common = (_stream(stream), m, n, _ptr(W0), _dtype(W0), _ptr(U), _ptr(Hbar))
    tail = (ctypes.byref(qcfg), ctypes.byref(bcfg) if bcfg is not None else None, _ptr(F), _ptr(F_next),
            _ptr(W_work), _ptr(adam_m), _ptr(adam_v), _ptr(bgd_disp), ctypes.byref(t), _ptr(codes), _ptr(scale),
            _ptr(zero), _ptr(W_deq), _dtype(W_deq) if W_deq is not None else REALQ_F32, int(block_begin),
            int(block_end), wp, wb)
    if block_loss is None:
        _check(lib().realq_quantize_layer(*common, _ptr(Dbar), _ptr(dead), *tail))
    else:
        _need(block_loss, torch.float32, (nb, 2), "block_loss")
        tp, tb = _ws(trace_ws)
        _check(lib().realq_quantize_layer_traced(*common, _ptr(dead), *tail, _ptr(block_loss), tp, tb))
    return t.value


def realq_quantize_grouped_workspace_size(m: int, n: int, n_row_groups: int, qcfg: QuantCfg,
                                          bcfg: Optional[BgdCfg] = None, has_F_next: bool = False,
                                          has_Dbar: bool = False) -> int:
    return int(lib().realq_quantize_grouped_workspace_size(m, n, n_row_groups, ctypes.byref(qcfg),
                                                           ctypes.byref(bcfg) if bcfg is not None else None,
                                                           int(has_F_next), int(has_Dbar)))


def realq_quantize_layer_grouped(W0: torch.Tensor, U_g: torch.Tensor, Hbar_g: Optional[torch.Tensor],
                                 dead_g: torch.Tensor, Hbar: Optional[torch.Tensor], qcfg: QuantCfg,
                                 W_work: torch.Tensor, codes: torch.Tensor, scale: torch.Tensor, zero: torch.Tensor, *,
                                 Dbar=None, bcfg: Optional[BgdCfg] = None, F=None, F_next=None, adam_m=None,
                                 adam_v=None, bgd_disp=None, adam_t: int = 0, W_deq=None, block_begin: int = 0,
                                 block_end: Optional[int] = None, ws=None, stream=None) -> int:
    """The sweep with row groups, group g against U_g[g]; returns the Adam step counter."""
    m, n = W0.shape
    ng = U_g.shape[0]
    nb = -(-n // qcfg.block_size)
    if block_end is None:
        block_end = nb
    _need(U_g, torch.float32, (ng, n, n), "U_g")
    _need(Hbar_g, torch.float32, (ng, n, n), "Hbar_g")
    _need(dead_g, torch.uint8, (ng, n), "dead_g")
    _need(W_work, torch.float32, (m, n), "W_work")
    _need(codes, torch.uint8, (m, (n + 1) // 2), "codes")
    _need(adam_m, torch.float32, (m, n), "adam_m")
    _need(adam_v, torch.float32, (m, n), "adam_v")
    _need(bgd_disp, torch.float32, (m, n), "bgd_disp")
    t = ctypes.c_int64(adam_t)
    wp, wb = _ws(ws)
    _check(lib().realq_quantize_layer_grouped(
        _stream(stream), m, n, _ptr(W0), _dtype(W0), ng, _ptr(U_g), _ptr(Hbar_g), _ptr(dead_g), _ptr(Hbar),
        _ptr(Dbar), ctypes.byref(qcfg), ctypes.byref(bcfg) if bcfg is not None else None, _ptr(F), _ptr(F_next),
        _ptr(W_work), _ptr(adam_m), _ptr(adam_v), _ptr(bgd_disp), ctypes.byref(t), _ptr(codes), _ptr(scale),
        _ptr(zero), _ptr(W_deq), _dtype(W_deq) if W_deq is not None else REALQ_F32, int(block_begin), int(block_end),
        wp, wb))
    return t.value


def realq_quantize_minibatch_workspace_size(m: int, n: int, n_minibatch: int, qcfg: QuantCfg,
                                            bcfg: Optional[BgdCfg] = None, has_F_next: bool = False) -> int:
    return int(lib().realq_quantize_minibatch_workspace_size(m, n, n_minibatch, ctypes.byref(qcfg),
                                                             ctypes.byref(bcfg) if bcfg is not None else None,
                                                             int(has_F_next)))


def realq_quantize_layer_minibatch(W0: torch.Tensor, U: torch.Tensor, Hbar: torch.Tensor, Hbar_mb: torch.Tensor,
                                   qcfg: QuantCfg, W_work: torch.Tensor, codes: torch.Tensor, scale: torch.Tensor,
                                   zero: torch.Tensor, *, dead=None, bcfg: Optional[BgdCfg] = None, F=None,
                                   F_next=None, adam_m=None, adam_v=None, bgd_disp=None, adam_t: int = 0, W_deq=None,
                                   block_begin: int = 0, block_end: Optional[int] = None, ws=None,
                                   stream=None) -> int:
    """The sweep with Block-GD steps on rotating calibration mini-batches; returns the Adam step counter."""
    m, n = W0.shape
    nmb = Hbar_mb.shape[0]
    if block_end is None:
        block_end = -(-n // qcfg.block_size)
    _need(Hbar_mb, torch.float32, (nmb, n, n), "Hbar_mb")
    _need(U, torch.float32, (n, n), "U")
    _need(W_work, torch.float32, (m, n), "W_work")
    _need(codes, torch.uint8, (m, (n + 1) // 2), "codes")
    for t_, nm in ((adam_m, "adam_m"), (adam_v, "adam_v"), (bgd_disp, "bgd_disp")):
        _need(t_, torch.float32, (m, n), nm)
    t = ctypes.c_int64(adam_t)
    wp, wb = _ws(ws)
    _check(lib().realq_quantize_layer_minibatch(
        _stream(stream), m, n, _ptr(W0), _dtype(W0), _ptr(U), _ptr(Hbar), _ptr(dead), nmb, _ptr(Hbar_mb),
        ctypes.byref(qcfg), ctypes.byref(bcfg) if bcfg is not None else None, _ptr(F), _ptr(F_next), _ptr(W_work),
        _ptr(adam_m), _ptr(adam_v), _ptr(bgd_disp), ctypes.byref(t), _ptr(codes), _ptr(scale), _ptr(zero),
        _ptr(W_deq), _dtype(W_deq) if W_deq is not None else REALQ_F32, int(block_begin), int(block_end), wp, wb))
    return t.value


def realq_quantize_tokens_workspace_size(m: int, n: int, T_mb: int, qcfg: QuantCfg, bcfg: Optional[BgdCfg] = None,
                                         has_F_next: bool = False) -> int:
    return int(lib().realq_quantize_tokens_workspace_size(m, n, int(T_mb), ctypes.byref(qcfg),
                                                          ctypes.byref(bcfg) if bcfg is not None else None,
                                                          int(has_F_next)))


def realq_quantize_layer_tokens(W0: torch.Tensor, U: torch.Tensor, Hbar: torch.Tensor, X_hat: torch.Tensor,
                                T_mb: int, a_loss_clip: float, qcfg: QuantCfg, W_work: torch.Tensor,
                                codes: torch.Tensor, scale: torch.Tensor, zero: torch.Tensor, *, dead=None,
                                bcfg: Optional[BgdCfg] = None, F=None, F_next=None, adam_m=None, adam_v=None,
                                bgd_disp=None, adam_t: int = 0, W_deq=None, block_begin: int = 0,
                                block_end: Optional[int] = None, ws=None, stream=None) -> int:
    """The sweep with Block-GD steps in token form on rotating mini-batches of
    X_hat's tokens, with per-token output clipping; returns the Adam step counter."""
    m, n = W0.shape
    T = X_hat.shape[0]
    if block_end is None:
        block_end = -(-n // qcfg.block_size)
    _need(X_hat, torch.bfloat16, (T, n), "X_hat")
    _need(U, torch.float32, (n, n), "U")
    _need(W_work, torch.float32, (m, n), "W_work")
    _need(codes, torch.uint8, (m, (n + 1) // 2), "codes")
    for t_, nm in ((adam_m, "adam_m"), (adam_v, "adam_v"), (bgd_disp, "bgd_disp")):
        _need(t_, torch.float32, (m, n), nm)
    t = ctypes.c_int64(adam_t)
    wp, wb = _ws(ws)
    _check(lib().realq_quantize_layer_tokens(
        _stream(stream), m, n, _ptr(W0), _dtype(W0), _ptr(U), _ptr(Hbar), _ptr(dead), _ptr(X_hat), T, int(T_mb),
        float(a_loss_clip), ctypes.byref(qcfg), ctypes.byref(bcfg) if bcfg is not None else None, _ptr(F),
        _ptr(F_next), _ptr(W_work), _ptr(adam_m), _ptr(adam_v), _ptr(bgd_disp), ctypes.byref(t), _ptr(codes),
        _ptr(scale), _ptr(zero), _ptr(W_deq), _dtype(W_deq) if W_deq is not None else REALQ_F32, int(block_begin),
        int(block_end), wp, wb))
    return t.value


def realq_bgd_workspace_size(m: int, n: int, has_F_next: bool = False, has_Dbar: bool = False) -> int:
    return int(lib().realq_bgd_workspace_size(m, n, int(has_F_next), int(has_Dbar)))


def realq_bgd_refine(W: torch.Tensor, W0: torch.Tensor, col_start: int, Hbar: torch.Tensor, F: torch.Tensor,
                     bcfg: BgdCfg, *, Dbar=None, F_next=None, alpha: float = 1.0, adam_m=None, adam_v=None,
                     adam_t: int = 0, ws=None, stream=None) -> int:
    m, n = W.shape
    t = ctypes.c_int64(adam_t)
    wp, wb = _ws(ws)
    _check(lib().realq_bgd_refine(_stream(stream), m, n, int(col_start), _ptr(W), _ptr(W0), _dtype(W0), _ptr(Hbar),
                                  _ptr(Dbar), _ptr(F), _ptr(F_next), float(alpha), _ptr(adam_m), _ptr(adam_v),
                                  ctypes.byref(t), ctypes.byref(bcfg), wp, wb))
    return t.value


def realq_surrogate_workspace_size(m: int, n: int) -> int:
    return int(lib().realq_surrogate_workspace_size(m, n))


def realq_surrogate_loss(W_hat: torch.Tensor, W0: torch.Tensor, Hbar: torch.Tensor, F: torch.Tensor,
                         loss_out: torch.Tensor, ws: torch.Tensor, stream=None):
    m, n = W_hat.shape
    wp, wb = _ws(ws)
    _check(lib().realq_surrogate_loss(_stream(stream), m, n, _ptr(W_hat), _ptr(W0), _dtype(W0), _ptr(Hbar), _ptr(F),
                                      _ptr(loss_out), wp, wb))


_BLOCK_KEYS = ("g1", "Wq", "Wk", "Wv", "Wo", "g2", "Wg", "Wu", "Wd")


def block_dims(d: int, n_heads: int, n_kv: int, head_dim: int, ffn: int, rms_eps: float = 1e-6,
               rope_base: float = 10000.0) -> BlockDims:
    return BlockDims(d, n_heads, n_kv, head_dim, ffn, rms_eps, rope_base)


def _block_shapes(dims: BlockDims) -> dict:
    d, qw, kw, f = dims.d, dims.n_heads * dims.head_dim, dims.n_kv * dims.head_dim, dims.ffn
    return {"g1": (d,), "Wq": (qw, d), "Wk": (kw, d), "Wv": (kw, d), "Wo": (d, qw), "g2": (d,), "Wg": (f, d),
            "Wu": (f, d), "Wd": (d, f)}


def _block_weights(w: dict, dims: Optional[BlockDims] = None) -> BlockWeights:
    """The C struct of a block's weights; with dims, every shape is checked
    (the library reads them at the sizes dims implies)."""
    shapes = _block_shapes(dims) if dims is not None else None
    for k in _BLOCK_KEYS:
        t = w[k]
        if t.dtype != torch.float32:
            raise ValueError(f"block weight {k}: expected float32, got {t.dtype}")
        if shapes is not None and tuple(t.shape) != shapes[k]:
            raise ValueError(f"block weight {k}: expected shape {shapes[k]}, got {tuple(t.shape)}")
    out = BlockWeights()
    for k in _BLOCK_KEYS:
        setattr(out, k, _ptr(w[k]).value)
    return out


def _need_tokens(x: Optional[torch.Tensor], dims: BlockDims, name: str, like: Optional[torch.Tensor] = None):
    if x is None:
        return
    if x.dim() != 3 or x.shape[2] != dims.d or x.dtype != torch.float32:
        raise ValueError(f"{name}: expected float32 (S, L, {dims.d}), got {x.dtype} {tuple(x.shape)}")
    if like is not None and x.shape != like.shape:
        raise ValueError(f"{name}: expected shape {tuple(like.shape)}, got {tuple(x.shape)}")


def realq_block_workspace_size(dims: BlockDims, S: int, L: int) -> int:
    return int(lib().realq_block_workspace_size(ctypes.byref(dims), int(S), int(L)))


def realq_set_tensor_tile(mode: int) -> None:
    """Output tile of the tf32x3 tensor-core products: 0 by grid (default),
    1 always 128 x 128, 2 always 128 x 256."""
    _check(lib().realq_set_tensor_tile(int(mode)))


def realq_set_quant_kernel(mode: int) -> None:
    """Kernel of the column-serial quantizer: 0 with block-wide barriers
    (default), 1 pipelined (identical results)."""
    _check(lib().realq_set_quant_kernel(int(mode)))


def realq_set_bgd_products(mode: int) -> None:
    """The plain Block-GD products: 1 f16x3 where m and n are multiples of 8
    (default), 0 tf32x3."""
    _check(lib().realq_set_bgd_products(int(mode)))


def realq_set_tensor_overlap(mode: int) -> None:
    """Wide-tile f16x3 products as persistent kernels with the epilogue
    overlapped: 1 the G product (default), 2 G and P, 0 none (one tile per
    CTA; identical results)."""
    _check(lib().realq_set_tensor_overlap(int(mode)))


def realq_set_block_attention(mode: int) -> None:
    """The block ops' attention: 1 tiled kernels (default), 0 one thread per
    row (the bodies of block_ops.cuh)."""
    _check(lib().realq_set_block_attention(int(mode)))


def realq_set_block_products(mode: int) -> None:
    """Products of the block ops: 0 fp32 CUDA-core tiles (default), 1 tf32x3
    tensor cores where the operands fit the workspace's plane scratch."""
    _check(lib().realq_set_block_products(int(mode)))


def realq_reverse_cosine_lr(i: int, L: int, lr_final: float) -> float:
    """The learning rate of decoder block i (1-based) of L: a reverse-cosine
    ramp from 0.01 lr_final at the first block to lr_final at the last."""
    out = ctypes.c_double(0.0)
    _check(lib().realq_reverse_cosine_lr(int(i), int(L), float(lr_final), ctypes.byref(out)))
    return out.value


def realq_block_forward(dims: BlockDims, weights: dict, x: torch.Tensor, y: torch.Tensor, ws: torch.Tensor,
                        stream=None):
    """y = block(x) for x, y of shape (S, L, d), fp32 (the decoder block of
    the exact sliding window)."""
    _need_tokens(x, dims, "x")
    S, L, d = x.shape
    _need(y, torch.float32, (S, L, d), "y")
    wp, wb = _ws(ws)
    w = _block_weights(weights, dims)
    _check(lib().realq_block_forward(_stream(stream), ctypes.byref(dims), ctypes.byref(w), S, L, _ptr(x), _ptr(y),
                                     wp, wb))


def realq_block_window(dims: BlockDims, weights: dict, h_ref: torch.Tensor, dh: torch.Tensor, F_next: torch.Tensor,
                       g_h: torch.Tensor, ws: torch.Tensor, loss: Optional[torch.Tensor] = None, stream=None):
    """The next block's Fisher loss (1/2T) sum_t dz_t^T F_next dz_t with
    dz = B(h_ref + dh) - B(h_ref), into loss (a 1-element fp32 tensor, or
    None), and its gradient in dh into g_h; all (S, L, d) fp32."""
    _need_tokens(h_ref, dims, "h_ref")
    S, L, d = h_ref.shape
    for t, name in ((dh, "dh"), (g_h, "g_h")):
        _need(t, torch.float32, (S, L, d), name)
    _need(F_next, torch.float32, (d, d), "F_next")
    wp, wb = _ws(ws)
    w = _block_weights(weights, dims)
    _check(lib().realq_block_window(_stream(stream), ctypes.byref(dims), ctypes.byref(w), S, L, _ptr(h_ref), _ptr(dh),
                                    _ptr(F_next), _ptr(g_h), _ptr(loss), wp, wb))


BLOCK_MODULES = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


def realq_block_module_workspace_size(dims: BlockDims, S: int, L: int, vocab: int = 0) -> int:
    return int(lib().realq_block_module_workspace_size(ctypes.byref(dims), int(S), int(L), int(vocab)))


def realq_block_head_workspace_size(d: int, S: int, L: int, vocab: int) -> int:
    return int(lib().realq_block_head_workspace_size(int(d), int(S), int(L), int(vocab)))


def realq_block_module_inputs(dims: BlockDims, weights: dict, x: torch.Tensor, module: str, X_out: torch.Tensor,
                              ws: torch.Tensor, stream=None):
    """The module's calibration inputs (S L x n) in a forward pass of the
    block with `weights` on x (S, L, d); ws as realq_block_forward."""
    _need_tokens(x, dims, "x")
    S, L, d = x.shape
    n = {"q_proj": d, "k_proj": d, "v_proj": d, "o_proj": dims.n_heads * dims.head_dim, "gate_proj": d,
         "up_proj": d, "down_proj": dims.ffn}[module]
    _need(X_out, torch.float32, (S * L, n), "X_out")
    wp, wb = _ws(ws)
    a = _block_weights(weights, dims)
    _check(lib().realq_block_module_inputs(_stream(stream), ctypes.byref(dims), ctypes.byref(a), S, L, _ptr(x),
                                           BLOCK_MODULES.index(module), _ptr(X_out), wp, wb))


def _opt_weights(w: Optional[dict], dims: Optional[BlockDims] = None):
    return ctypes.byref(_block_weights(w, dims)) if w is not None else None


_MODULE_KEY = {"q_proj": "Wq", "k_proj": "Wk", "v_proj": "Wv", "o_proj": "Wo", "gate_proj": "Wg", "up_proj": "Wu",
               "down_proj": "Wd"}


def _need_module(dims: BlockDims, module: str, x: torch.Tensor, x_hat: Optional[torch.Tensor],
                 W_module: Optional[torch.Tensor], Fs=()):
    # the shapes the library reads: tokens (S, L, d), x_hat like x, the
    # module's weight as dims implies, d x d Fishers
    _need_tokens(x, dims, "x")
    _need_tokens(x_hat, dims, "x_hat", like=x)
    _need(W_module, torch.float32, _block_shapes(dims)[_MODULE_KEY[module]], "W_module")
    for F, name in Fs:
        _need(F, torch.float32, (dims.d, dims.d), name)


def realq_block_module_window(dims: BlockDims, this_block: dict, next_block: dict, x: torch.Tensor, module: str,
                              W_module: torch.Tensor, alpha: float, F_this: torch.Tensor, F_next: torch.Tensor,
                              grad: torch.Tensor, ws: torch.Tensor, loss: Optional[torch.Tensor] = None,
                              this_block_hat: Optional[dict] = None, x_hat: Optional[torch.Tensor] = None,
                              stream=None):
    """The exact two-block window of one module of block l: its loss into
    loss (or None) and its gradient in W_module into grad (W_module's shape).
    this_block_hat / x_hat: block l's weights and input in the current pass
    (the model quantized so far); None: the reference ones."""
    _need_module(dims, module, x, x_hat, W_module, ((F_this, "F_this"), (F_next, "F_next")))
    S, L, d = x.shape
    _need(grad, torch.float32, tuple(W_module.shape), "grad")
    wp, wb = _ws(ws)
    a, b = _block_weights(this_block, dims), _block_weights(next_block, dims)
    _check(lib().realq_block_module_window(_stream(stream), ctypes.byref(dims), ctypes.byref(a),
                                           _opt_weights(this_block_hat, dims), ctypes.byref(b), S, L, _ptr(x),
                                           _ptr(x_hat),
                                           BLOCK_MODULES.index(module), _ptr(W_module), float(alpha), _ptr(F_this),
                                           _ptr(F_next), _ptr(grad), _ptr(loss), wp, wb))


def realq_block_head_kl(gf: torch.Tensor, Wh: torch.Tensor, h_ref: torch.Tensor, dh: torch.Tensor,
                        g_h: torch.Tensor, ws: torch.Tensor, loss: Optional[torch.Tensor] = None,
                        rms_eps: float = 1e-6, stream=None):
    """The final block's KL at the LM head between the outputs h_ref and
    h_ref + dh, and its gradient in dh; h_ref, dh, g_h (S, L, d) fp32."""
    S, L, d = h_ref.shape
    V = Wh.shape[0]
    _need(g_h, torch.float32, (S, L, d), "g_h")
    wp, wb = _ws(ws)
    _check(lib().realq_block_head_kl(_stream(stream), d, S, L, _ptr(gf), _ptr(Wh), V, float(rms_eps), _ptr(h_ref),
                                     _ptr(dh), _ptr(g_h), _ptr(loss), wp, wb))


def realq_block_module_kl(dims: BlockDims, this_block: dict, x: torch.Tensor, module: str, W_module: torch.Tensor,
                          gf: torch.Tensor, Wh: torch.Tensor, grad: torch.Tensor, ws: torch.Tensor,
                          loss: Optional[torch.Tensor] = None, this_block_hat: Optional[dict] = None,
                          x_hat: Optional[torch.Tensor] = None, stream=None):
    """The final block's KL for one module's weight, and its gradient
    (this_block_hat / x_hat as for realq_block_module_window)."""
    _need_module(dims, module, x, x_hat, W_module)
    _need(Wh, torch.float32, (Wh.shape[0], dims.d), "Wh")
    _need(gf, torch.float32, (dims.d,), "gf")
    S, L, d = x.shape
    _need(grad, torch.float32, tuple(W_module.shape), "grad")
    wp, wb = _ws(ws)
    a = _block_weights(this_block, dims)
    _check(lib().realq_block_module_kl(_stream(stream), ctypes.byref(dims), ctypes.byref(a),
                                       _opt_weights(this_block_hat, dims), S, L, _ptr(x), _ptr(x_hat),
                                       BLOCK_MODULES.index(module), _ptr(W_module), _ptr(gf), _ptr(Wh), Wh.shape[0],
                                       _ptr(grad), _ptr(loss), wp, wb))


def realq_quantize_window_workspace_size(dims: BlockDims, S: int, L: int, module: str, qcfg: QuantCfg,
                                         vocab: int = 0) -> int:
    """Workspace bytes of realq_quantize_layer_window (vocab 0: the exact
    window; the LM head's vocabulary: the final block's KL)."""
    return int(lib().realq_quantize_window_workspace_size(ctypes.byref(dims), int(S), int(L),
                                                          BLOCK_MODULES.index(module), int(vocab),
                                                          ctypes.byref(qcfg)))


def realq_quantize_layer_window(dims: BlockDims, this_block: dict, next_block: Optional[dict], x: torch.Tensor,
                                module: str, U: torch.Tensor, qcfg: QuantCfg, bcfg: BgdCfg, W_work: torch.Tensor,
                                codes: torch.Tensor, scale: torch.Tensor, zero: torch.Tensor, *, F_this=None,
                                F_next=None, head_gf=None, head_Wh=None, dead=None, adam_m=None, adam_v=None,
                                adam_t: int = 0, W_deq=None, block_loss: Optional[torch.Tensor] = None,
                                block_begin: int = 0, block_end: Optional[int] = None, ws=None,
                                this_block_hat: Optional[dict] = None, x_hat: Optional[torch.Tensor] = None,
                                n_minibatch: int = 1, stream=None) -> int:
    """The column sweep of one module of decoder block l with Block-GD on the
    exact two-block window (next_block given, with F_this and F_next) or on
    the final block's KL at the LM head (next_block None, with head_gf and
    head_Wh); x (S, L, d) is block l's input.  The module's weight in
    this_block is the reference and the sweep's W0; this_block_hat / x_hat
    are block l's weights and input in the current pass (the model quantized
    so far; None: the reference ones).  With n_minibatch > 1, x and x_hat
    hold that many calibration mini-batches of whole sequences, and each
    Block-GD step takes one in rotation.  Runs blocks [block_begin,
    block_end); returns the optimizer step counter."""
    _need_module(dims, module, x, x_hat, None, ((F_this, "F_this"), (F_next, "F_next")))
    if head_Wh is not None:
        _need(head_Wh, torch.float32, (head_Wh.shape[0], dims.d), "head_Wh")
        _need(head_gf, torch.float32, (dims.d,), "head_gf")
    S_all, L, d = x.shape
    if n_minibatch < 1 or S_all % n_minibatch:
        raise ValueError(f"{S_all} sequences do not split into {n_minibatch} mini-batches")
    S = S_all // n_minibatch
    Wref = this_block[{"q_proj": "Wq", "k_proj": "Wk", "v_proj": "Wv", "o_proj": "Wo", "gate_proj": "Wg",
                       "up_proj": "Wu", "down_proj": "Wd"}[module]]
    m, n = Wref.shape
    nb = -(-n // qcfg.block_size)
    if block_end is None:
        block_end = nb
    _need(W_work, torch.float32, (m, n), "W_work")
    _need(U, torch.float32, (n, n), "U")
    _need(codes, torch.uint8, (m, (n + 1) // 2), "codes")
    _need(adam_m, torch.float32, (m, n), "adam_m")
    _need(adam_v, torch.float32, (m, n), "adam_v")
    _need(block_loss, torch.float32, (nb, 2), "block_loss")
    t = ctypes.c_int64(adam_t)
    wp, wb = _ws(ws)
    a = _block_weights(this_block, dims)
    b = _block_weights(next_block, dims) if next_block is not None else None
    V = int(head_Wh.shape[0]) if head_Wh is not None else 0
    _check(lib().realq_quantize_layer_window(
        _stream(stream), ctypes.byref(dims), ctypes.byref(a), _opt_weights(this_block_hat, dims),
        ctypes.byref(b) if b is not None else None, S, L, int(n_minibatch), _ptr(x), _ptr(x_hat),
        BLOCK_MODULES.index(module),
        _ptr(F_this), _ptr(F_next), _ptr(head_gf), _ptr(head_Wh), V,
        _ptr(U), _ptr(dead), ctypes.byref(qcfg), ctypes.byref(bcfg), _ptr(W_work), _ptr(adam_m), _ptr(adam_v),
        ctypes.byref(t), _ptr(codes), _ptr(scale), _ptr(zero), _ptr(W_deq),
        _dtype(W_deq) if W_deq is not None else REALQ_F32, _ptr(block_loss), int(block_begin), int(block_end), wp,
        wb))
    return t.value


def realq_workspace_status(ws: torch.Tensor, stream=None) -> int:
    """Synchronizes; raises RealqError if the sweep recorded a non-finite weight."""
    wp, wb = _ws(ws)
    _check(lib().realq_workspace_status(_stream(stream), wp, wb))
    return REALQ_OK


def realq_status_string(status: int) -> str:
    return lib().realq_status_string(status).decode()


def realq_last_error() -> str:
    return lib().realq_last_error().decode(errors="replace")


def realq_launch_count() -> int:
    return int(lib().realq_launch_count())


def realq_profile_enable(on: bool = True):
    lib().realq_profile_enable(int(on))


def realq_profile_collect(max_entries: int = 64) -> dict:
    """{kernel name: (launches, total_ms)} since the last collect (synchronizes the recorded events)."""
    arr = (KernelStat * max_entries)()
    k = lib().realq_profile_collect(arr, max_entries)
    return {arr[i].name.decode(): (int(arr[i].launches), float(arr[i].total_ms)) for i in range(k)}
