"""Thin Python binding of libsgdkv (include/sgdkv.h), same names as the C-ABI.

Argument marshalling only: every step of the compression path runs in the CUDA library.
Tensors are torch tensors (device memory, caller-owned); host arrays are NumPy.  If the
library has not been built, every call raises ``LibraryMissing``; there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "lib", "libsgdkv.so")

OK, ERR_INVALID_ARG, ERR_INFEASIBLE_BUDGET, ERR_WORKSPACE, ERR_CUDA, ERR_TIMEOUT, \
    ERR_UNSUPPORTED, ERR_INTERNAL = range(8)
ALLOC_GREEDY, ALLOC_PROPORTIONAL, ALLOC_THRESHOLD, ALLOC_REVERSE = 0, 1, 2, 3
EXPORTED = ("sgdkv_status_string", "sgdkv_version", "sgdkv_allocate_budgets",
            "sgdkv_workspace_bytes", "sgdkv_score", "sgdkv_compact", "sgdkv_compress_layer",
            "sgdkv_last_error", "sgdkv_launch_count", "sgdkv_debug_set_score_hooks",
            "sgdkv_last_cuda_error_string", "sgdkv_score_static",
            "sgdkv_debug_enable_kernel_timing", "sgdkv_debug_kernel_timing", "sgdkv_score_ex",
            "sgdkv_mix_head_scores", "sgdkv_score_raw", "sgdkv_pool_raw",
            "sgdkv_window_stats", "sgdkv_window_sums", "sgdkv_pool_compact",
            "sgdkv_decode_workspace_bytes", "sgdkv_decode_attention")


class LibraryMissing(RuntimeError):
    pass


class SgdkvError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = f"{where}: {status_string(status)} (status {status})"
        if status == ERR_CUDA:
            msg += ": " + lib().sgdkv_last_cuda_error_string().decode()
        super().__init__(msg)


_lib = None
_P = ctypes.c_void_p
_I32, _I64, _SZ = ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t


def lib():
    """The loaded libsgdkv.so (loaded once)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise LibraryMissing(f"{LIB_PATH} not built: run `python -c \"import __graft_entry__ as g; g.build()\"`")
        L = ctypes.CDLL(LIB_PATH)
        L.sgdkv_status_string.restype = ctypes.c_char_p
        L.sgdkv_status_string.argtypes = [ctypes.c_int]
        L.sgdkv_version.restype = ctypes.c_int
        L.sgdkv_allocate_budgets.restype = ctypes.c_int
        L.sgdkv_allocate_budgets.argtypes = [_P, _I32, _I64, _I64, _I64, _I32, _P]
        L.sgdkv_mix_head_scores.restype = ctypes.c_int
        L.sgdkv_mix_head_scores.argtypes = [_P, _P, _I32, _P]
        L.sgdkv_workspace_bytes.restype = _SZ
        L.sgdkv_workspace_bytes.argtypes = [_I32, _I32, _I64, _I32, _I32]
        L.sgdkv_score.restype = ctypes.c_int
        L.sgdkv_score.argtypes = [_P, _P, _I32, _I32, _I64, _I32, _I32, _I32, _P, _P, _SZ, _P]
        L.sgdkv_compact.restype = ctypes.c_int
        L.sgdkv_compact.argtypes = [_P, _P, _P, _P, _I32, _I64, _I32, _I64, _I64, _P, _P, _P, _P,
                                    _P, _SZ, _P]
        L.sgdkv_compress_layer.restype = ctypes.c_int
        L.sgdkv_compress_layer.argtypes = [_P, _P, _P, _P, _I32, _I32, _I64, _I32, _I32, _I32,
                                           _I64, _I64, _P, _P, _P, _P, _P, _P, _SZ, _P]
        L.sgdkv_last_error.restype = ctypes.c_int
        L.sgdkv_last_error.argtypes = [_P, _P]
        L.sgdkv_launch_count.restype = ctypes.c_uint64
        L.sgdkv_last_cuda_error_string.restype = ctypes.c_char_p
        L.sgdkv_score_ex.restype = ctypes.c_int
        L.sgdkv_score_ex.argtypes = [_P, _P, _I32, _I32, _I64, _I32, _I32, _I32, ctypes.c_uint32,
                                     _P, _P, _P, _SZ, _P]
        L.sgdkv_score_raw.restype = ctypes.c_int
        L.sgdkv_score_raw.argtypes = [_P, _P, _I32, _I32, _I64, _I32, _I32, ctypes.c_uint32, _P,
                                      _P, _SZ, _P]
        for fn in (L.sgdkv_window_stats, L.sgdkv_window_sums):
            fn.restype = ctypes.c_int
            fn.argtypes = [_P, _P, _I32, _I32, _I64, _I32, _I32, ctypes.c_uint32, _P, _P, _SZ, _P]
        L.sgdkv_pool_raw.restype = ctypes.c_int
        L.sgdkv_pool_raw.argtypes = [_P, _SZ, _I32, _I64, _I32, ctypes.c_uint32, _P, _P]
        L.sgdkv_decode_workspace_bytes.restype = _SZ
        L.sgdkv_decode_workspace_bytes.argtypes = [_I32, _I32, _I32, _I32, _I64]
        L.sgdkv_decode_attention.restype = ctypes.c_int
        L.sgdkv_decode_attention.argtypes = [_P, _I32, _I32, _I32, _I32, _P, _P, _P, _P, _P,
                                             _SZ, _P]
        L.sgdkv_pool_compact.restype = ctypes.c_int
        L.sgdkv_pool_compact.argtypes = [_P, _SZ, _I32, ctypes.c_uint32, _P, _P, _P, _I32, _I64,
                                         _I32, _I64, _I64, _P, _P, _P, _P, _P, _P, _SZ, _P]
        L.sgdkv_score_static.restype = ctypes.c_int
        L.sgdkv_score_static.argtypes = [_P, _P, _I32, _I32, _I64, _I32, _I32, _I32, _P, _P, _P]
        L.sgdkv_debug_set_score_hooks.restype = None
        L.sgdkv_debug_set_score_hooks.argtypes = [ctypes.c_uint32, ctypes.c_uint64]
        L.sgdkv_debug_enable_kernel_timing.restype = None
        L.sgdkv_debug_enable_kernel_timing.argtypes = [ctypes.c_uint32]
        L.sgdkv_debug_kernel_timing.restype = ctypes.c_int
        L.sgdkv_debug_kernel_timing.argtypes = [ctypes.c_int, ctypes.POINTER(ctypes.c_double),
                                                ctypes.POINTER(ctypes.c_int64)]
        _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().sgdkv_status_string(int(status)).decode()


def _check(status: int, where: str):
    if status != OK:
        raise SgdkvError(status, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(int(getattr(stream, "cuda_stream", stream)))


def sgdkv_version() -> int:
    return lib().sgdkv_version()


def sgdkv_allocate_budgets(head_scores, context_len: int, total_budget: int, floor: int,
                           mode: int = ALLOC_GREEDY) -> np.ndarray:
    s = np.ascontiguousarray(head_scores, dtype=np.float32)
    out = np.zeros(s.size, dtype=np.int64)
    st = lib().sgdkv_allocate_budgets(s.ctypes.data_as(_P), s.size, int(context_len),
                                      int(total_budget), int(floor), int(mode),
                                      out.ctypes.data_as(_P))
    _check(st, "sgdkv_allocate_budgets")
    return out


def sgdkv_mix_head_scores(a, b) -> np.ndarray:
    """SGD-KV + HeadKV head scores: the mean of the two normalised score sets."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    b = np.ascontiguousarray(b, dtype=np.float32)
    if a.size != b.size:
        raise ValueError("score sets differ in length")
    out = np.zeros(a.size, dtype=np.float32)
    st = lib().sgdkv_mix_head_scores(a.ctypes.data_as(_P), b.ctypes.data_as(_P), a.size,
                                     out.ctypes.data_as(_P))
    _check(st, "sgdkv_mix_head_scores")
    return out


def sgdkv_workspace_bytes(Hq: int, Hkv: int, L: int, d: int, W: int) -> int:
    return int(lib().sgdkv_workspace_bytes(Hq, Hkv, L, d, W))


def make_workspace(Hq: int, Hkv: int, L: int, W: int, device="cuda", d: int = 128):
    """Zero-filled workspace tensor for this shape (caller-owned device memory)."""
    import torch
    n = sgdkv_workspace_bytes(Hq, Hkv, L, d, W)
    if n == 0:
        raise SgdkvError(ERR_UNSUPPORTED, "sgdkv_workspace_bytes")
    return torch.zeros(n, dtype=torch.uint8, device=device)


SCORE_PROXY_QUERY = 1
SCORE_AGG_SUM, SCORE_AGG_IPT_MAX, SCORE_AGG_IPT_MEAN, SCORE_AGG_IPT_ONLY = 0, 2, 4, 6
SCORE_DETERMINISTIC = 8


def sgdkv_score(q_win, K, W: int, pool: int, scores_out, workspace, stream=None, flags: int = 0,
                head_weights=None):
    """Window scores (flags 0: causal observation window, summed over the GQA group) or,
    through sgdkv_score_ex, SCORE_PROXY_QUERY (external queries that see every key) and the
    SCORE_AGG_IPT_* group aggregations (head_weights: device fp32 [Hq])."""
    Hq, W_, d = q_win.shape
    Hkv, L, _ = K.shape
    if flags == 0 and head_weights is None:
        st = lib().sgdkv_score(_ptr(q_win), _ptr(K), Hq, Hkv, L, d, W, pool, _ptr(scores_out),
                               _ptr(workspace), workspace.numel(), _stream(stream))
        _check(st, "sgdkv_score")
        return
    st = lib().sgdkv_score_ex(_ptr(q_win), _ptr(K), Hq, Hkv, L, d, W, pool, int(flags),
                              _ptr(head_weights), _ptr(scores_out), _ptr(workspace),
                              workspace.numel(), _stream(stream))
    _check(st, "sgdkv_score_ex")


def sgdkv_score_raw(q_win, K, W: int, workspace, stream=None, flags: int = 0, head_weights=None):
    """Both scoring passes; the raw window scores stay in the workspace for sgdkv_pool_raw."""
    Hq, _, d = q_win.shape
    Hkv, L, _ = K.shape
    st = lib().sgdkv_score_raw(_ptr(q_win), _ptr(K), Hq, Hkv, L, d, W, int(flags),
                               _ptr(head_weights), _ptr(workspace), workspace.numel(),
                               _stream(stream))
    _check(st, "sgdkv_score_raw")


def _window_pass(fn, name, q_win, K, W, workspace, stream, flags, head_weights):
    Hq, _, d = q_win.shape
    Hkv, L, _ = K.shape
    st = fn(_ptr(q_win), _ptr(K), Hq, Hkv, L, d, W, int(flags), _ptr(head_weights),
            _ptr(workspace), workspace.numel(), _stream(stream))
    _check(st, name)


def sgdkv_window_stats(q_win, K, W: int, workspace, stream=None, flags: int = 0,
                       head_weights=None):
    """Pass 1 of the scoring: per-window-row softmax statistics into the workspace."""
    _window_pass(lib().sgdkv_window_stats, "sgdkv_window_stats", q_win, K, W, workspace, stream,
                 flags, head_weights)


def sgdkv_window_sums(q_win, K, W: int, workspace, stream=None, flags: int = 0,
                      head_weights=None):
    """Pass 2 of the scoring: the raw window scores, from sgdkv_window_stats' statistics."""
    _window_pass(lib().sgdkv_window_sums, "sgdkv_window_sums", q_win, K, W, workspace, stream,
                 flags, head_weights)


def sgdkv_pool_raw(workspace, Hkv: int, L: int, pool: int, scores_out, stream=None,
                   flags: int = 0):
    """Max-pool of the raw window scores a sgdkv_score_raw call left in the workspace."""
    st = lib().sgdkv_pool_raw(_ptr(workspace), workspace.numel(), int(Hkv), int(L), int(pool),
                              int(flags), _ptr(scores_out), _stream(stream))
    _check(st, "sgdkv_pool_raw")


def sgdkv_score_static(q_win, K, W: int, pool: int, scores_out, status_out=None, stream=None):
    """sgdkv_score with the library's static scratch instead of a caller workspace."""
    Hq, _, d = q_win.shape
    Hkv, L, _ = K.shape
    st = lib().sgdkv_score_static(_ptr(q_win), _ptr(K), Hq, Hkv, L, d, W, pool,
                                  _ptr(scores_out), _ptr(status_out), _stream(stream))
    _check(st, "sgdkv_score_static")


def _budgets(b):
    return np.ascontiguousarray(b, dtype=np.int64)


def sgdkv_compact(K, V, scores, budgets, n_sink: int, n_recent: int, indices_out,
                  cu_seqlens_out, K_out, V_out, workspace, stream=None):
    Hkv, L, d = K.shape
    b = _budgets(budgets)
    st = lib().sgdkv_compact(_ptr(K), _ptr(V), _ptr(scores), b.ctypes.data_as(_P), Hkv, L, d,
                             n_sink, n_recent, _ptr(indices_out), _ptr(cu_seqlens_out),
                             _ptr(K_out), _ptr(V_out), _ptr(workspace), workspace.numel(),
                             _stream(stream))
    _check(st, "sgdkv_compact")


def sgdkv_pool_compact(score_workspace, pool: int, K, V, budgets, n_sink: int, n_recent: int,
                       scores_out, indices_out, cu_seqlens_out, K_out, V_out, workspace,
                       stream=None, flags: int = 0):
    """sgdkv_pool_raw + sgdkv_compact in one call, from the raw scores in score_workspace."""
    Hkv, L, d = K.shape
    b = _budgets(budgets)
    st = lib().sgdkv_pool_compact(_ptr(score_workspace), score_workspace.numel(), int(pool),
                                  int(flags), _ptr(K), _ptr(V), b.ctypes.data_as(_P), Hkv, L,
                                  d, n_sink, n_recent, _ptr(scores_out), _ptr(indices_out),
                                  _ptr(cu_seqlens_out), _ptr(K_out), _ptr(V_out),
                                  _ptr(workspace), workspace.numel(), _stream(stream))
    _check(st, "sgdkv_pool_compact")


def sgdkv_decode_workspace_bytes(Hq: int, Hkv: int, n_tok: int, d: int, total_rows: int) -> int:
    return int(lib().sgdkv_decode_workspace_bytes(int(Hq), int(Hkv), int(n_tok), int(d),
                                                  int(total_rows)))


def make_decode_workspace(Hq: int, Hkv: int, n_tok: int, total_rows: int, device="cuda",
                          d: int = 128):
    """Workspace tensor for sgdkv_decode_attention (caller-owned device memory)."""
    import torch
    n = sgdkv_decode_workspace_bytes(Hq, Hkv, n_tok, d, total_rows)
    if n == 0:
        raise SgdkvError(ERR_UNSUPPORTED, "sgdkv_decode_workspace_bytes")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def sgdkv_decode_attention(q, K_cache, V_cache, budgets, out, workspace, stream=None):
    """Attention of q [Hq][n_tok][d] over the compressed cache; out fp32 [Hq][n_tok][d]."""
    Hq, n_tok, d = q.shape
    b = _budgets(budgets)
    st = lib().sgdkv_decode_attention(_ptr(q), Hq, len(b), n_tok, d, _ptr(K_cache),
                                      _ptr(V_cache), b.ctypes.data_as(_P), _ptr(out),
                                      _ptr(workspace), workspace.numel(), _stream(stream))
    _check(st, "sgdkv_decode_attention")


def sgdkv_compress_layer(q_win, K, V, budgets, W: int, pool: int, n_sink: int, n_recent: int,
                         scores_out, indices_out, cu_seqlens_out, K_out, V_out, workspace,
                         stream=None):
    Hq, _, d = q_win.shape
    Hkv, L, _ = K.shape
    b = _budgets(budgets)
    st = lib().sgdkv_compress_layer(_ptr(q_win), _ptr(K), _ptr(V), b.ctypes.data_as(_P), Hq,
                                    Hkv, L, d, W, pool, n_sink, n_recent, _ptr(scores_out),
                                    _ptr(indices_out), _ptr(cu_seqlens_out), _ptr(K_out),
                                    _ptr(V_out), _ptr(workspace), workspace.numel(),
                                    _stream(stream))
    _check(st, "sgdkv_compress_layer")


def sgdkv_launch_count() -> int:
    return int(lib().sgdkv_launch_count())


def sgdkv_debug_set_score_hooks(flags: int, wait_ns: int = 0) -> None:
    lib().sgdkv_debug_set_score_hooks(int(flags), int(wait_ns))


KERNEL_SCORE_PASS1, KERNEL_SCORE_PASS2, KERNEL_POOL, KERNEL_SELECT, KERNEL_GATHER, \
    KERNEL_DECODE = range(6)


def sgdkv_debug_enable_kernel_timing(kinds=()) -> None:
    """Times every launch of the given kernel kinds (an empty set turns timing off)."""
    mask = 0
    for k in kinds:
        mask |= 1 << int(k)
    lib().sgdkv_debug_enable_kernel_timing(mask)


def sgdkv_debug_kernel_timing(kind: int):
    """(summed milliseconds, launches) of the kernels of one kind timed since the last call."""
    ms, n = ctypes.c_double(0.0), ctypes.c_int64(0)
    st = lib().sgdkv_debug_kernel_timing(int(kind), ctypes.byref(ms), ctypes.byref(n))
    if st != OK:
        raise SgdkvError(st, "sgdkv_debug_kernel_timing")
    return ms.value, n.value


def sgdkv_last_error(workspace, stream=None) -> int:
    return int(lib().sgdkv_last_error(_ptr(workspace), _stream(stream)))


def compress_layer_alloc(q_win, K, V, budgets, W: int, pool: int, n_sink: int, n_recent: int,
                         workspace, stream=None, want_scores: bool = True):
    """Allocates the outputs with torch, calls sgdkv_compress_layer, returns them."""
    import torch
    Hkv, L, d = K.shape
    total = int(np.sum(_budgets(budgets)))
    dev = K.device
    scores = torch.empty((Hkv, L), dtype=torch.float32, device=dev) if want_scores else None
    idx = torch.empty(max(total, 1), dtype=torch.int32, device=dev)
    cu = torch.empty(Hkv + 1, dtype=torch.int32, device=dev)
    ko = torch.empty((max(total, 1), d), dtype=K.dtype, device=dev)
    vo = torch.empty((max(total, 1), d), dtype=V.dtype, device=dev)
    sgdkv_compress_layer(q_win, K, V, budgets, W, pool, n_sink, n_recent, scores, idx, cu, ko,
                         vo, workspace, stream)
    return dict(scores=scores, indices=idx[:total], cu_seqlens=cu, K_out=ko[:total],
                V_out=vo[:total])
