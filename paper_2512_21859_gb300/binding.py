"""Thin ctypes binding of libtimebill_kv.so (C ABI: include/timebill_kv.h).

Argument marshalling only: the functions below carry the C entry points'
names, turn tensors into device pointers and host lists into the
descriptor structs, and raise ``TbError`` on a non-OK status. Every step of
the computation runs in the library's CUDA kernels. Device buffers may be
torch tensors (their data_ptr() is passed) or plain integer addresses.
If the library has not been built, the first call raises RuntimeError.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

__all__ = [
    "TB_OK", "TB_ERR_INVALID_ARG", "TB_ERR_UNSUPPORTED", "TB_ERR_WORKSPACE",
    "TB_ERR_CUDA", "TB_ERR_TIMEOUT", "TB_F32", "TB_BF16", "TB_MAX_BATCH",
    "TbError", "EvictDesc", "DecodeDesc", "library_path", "load",
    "tb_status_string", "tb_abi_version", "tb_last_error_detail", "tb_launch_counter",
    "tb_retained_count", "tb_retained_count_ex", "TB_EVICT_BUDGET_INCLUDES_WINDOW",
    "TB_EVICT_AVG_POOL", "TB_EVICT_GATHER_CONCURRENT", "TB_DECODE_EARLY_CACHE_READ", "TB_DECODE_CONCURRENT", "tb_evict_layout",
    "tb_evict_workspace_size", "tb_window_scores", "tb_window_scores_lse", "tb_select_topk",
    "tb_select_ctas", "tb_gather_kv", "tb_score_evict",
    "tb_decode_workspace_size", "tb_decode_attn", "tb_read_status",
    "tb_decode_attn_noalloc", "tb_decode_noalloc_status", "TB_NOALLOC_SCRATCH_BYTES", "tb_diag_bounded_wait",
    "tb_decode_workspace_prepare", "tb_decode_attn_prepared",
    "TimeModel", "tb_wcet", "tb_alpha_star", "tb_fit_time_model",
]

TB_OK, TB_ERR_INVALID_ARG, TB_ERR_UNSUPPORTED, TB_ERR_WORKSPACE, TB_ERR_CUDA, TB_ERR_TIMEOUT = range(6)
TB_F32, TB_BF16 = 0, 1
TB_EVICT_BUDGET_INCLUDES_WINDOW, TB_EVICT_AVG_POOL, TB_EVICT_GATHER_CONCURRENT = 1, 2, 4
TB_DECODE_EARLY_CACHE_READ, TB_DECODE_CONCURRENT = 1, 2
TB_MAX_BATCH = 64
TB_NOALLOC_SCRATCH_BYTES = 4 << 20

_I64P = ctypes.POINTER(ctypes.c_int64)
_F64P = ctypes.POINTER(ctypes.c_double)


class _EvictDescC(ctypes.Structure):
    _fields_ = [
        ("batch", ctypes.c_int32), ("hq", ctypes.c_int32), ("hkv", ctypes.c_int32),
        ("head_dim", ctypes.c_int32), ("window", ctypes.c_int32), ("pool_k", ctypes.c_int32),
        ("dtype", ctypes.c_int32), ("flags", ctypes.c_int32),
        ("n", _I64P), ("alpha", _F64P), ("kv_offset", _I64P), ("kv_rows", ctypes.c_int64),
        ("out_offset", _I64P), ("out_cap", _I64P), ("out_rows", ctypes.c_int64),
    ]


class _DecodeDescC(ctypes.Structure):
    _fields_ = [
        ("batch", ctypes.c_int32), ("hq", ctypes.c_int32), ("hkv", ctypes.c_int32),
        ("head_dim", ctypes.c_int32), ("dtype", ctypes.c_int32), ("out_dtype", ctypes.c_int32),
        ("cache_offset", _I64P), ("cache_cap", _I64P), ("cache_rows", ctypes.c_int64),
        ("max_len", ctypes.c_int64), ("flags", ctypes.c_int32), ("max_ctas", ctypes.c_int32),
    ]


class TbError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        detail = ""
        if status == TB_ERR_CUDA:
            try:
                detail = ": " + tb_last_error_detail()
            except Exception:  # pragma: no cover
                pass
        super().__init__("%s failed: %s (status %d)%s" % (where, tb_status_string(status), status, detail))


def library_path() -> str:
    """The release library, or with TB_LIBRARY=debug the TB_DEBUG build
    (libtimebill_kv_debug.so, built by build.build(debug=True))."""
    name = "libtimebill_kv_debug.so" if os.environ.get("TB_LIBRARY") == "debug" else "libtimebill_kv.so"
    return os.path.join(os.path.dirname(os.path.abspath(__file__)), name)


_LIB = None


def load():
    """Loads the shared library (once) and declares the entry points."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = library_path()
    if not os.path.exists(path):
        raise RuntimeError("libtimebill_kv.so is not built (expected at %s); run "
                           "paper_2512_21859_gb300.build.build()" % path)
    lib = ctypes.CDLL(path)
    P = ctypes.c_void_p
    I = ctypes.c_int32
    SZ = ctypes.c_size_t
    sig = {
        "tb_status_string": (ctypes.c_char_p, [I]),
        "tb_abi_version": (I, []),
        "tb_last_error_detail": (ctypes.c_char_p, []),
        "tb_launch_counter": (ctypes.c_uint64, []),
        "tb_retained_count": (I, [ctypes.c_int64, I, ctypes.c_double, _I64P, _I64P]),
        "tb_retained_count_ex": (I, [ctypes.c_int64, I, ctypes.c_double, I, _I64P, _I64P]),
        "tb_evict_layout": (I, [P, _I64P, _I64P]),
        "tb_evict_workspace_size": (I, [P, ctypes.POINTER(SZ)]),
        "tb_window_scores": (I, [P, P, P, P, P, SZ, P]),
        "tb_window_scores_lse": (I, [P, P, P, P, P, P, SZ, P]),
        "tb_select_topk": (I, [P, P, P, P, P, SZ, P]),
        "tb_select_ctas": (I, [P, ctypes.POINTER(I)]),
        "tb_gather_kv": (I, [P, P, P, P, P, P, P]),
        "tb_score_evict": (I, [P, P, P, P, P, P, P, P, P, SZ, P]),
        "tb_decode_workspace_size": (I, [P, ctypes.POINTER(SZ)]),
        "tb_decode_attn": (I, [P, P, P, P, P, P, P, SZ, P]),
        "tb_read_status": (I, [P, SZ, P, ctypes.POINTER(I)]),
        "tb_decode_attn_noalloc": (I, [P, P, P, P, P, P, P]),
        "tb_decode_noalloc_status": (I, [P, ctypes.POINTER(I)]),
        "tb_decode_workspace_prepare": (I, [P, P, SZ, P]),
        "tb_decode_attn_prepared": (I, [P, P, P, P, P, P, P, SZ, P]),
        "tb_diag_bounded_wait": (I, [P, SZ, ctypes.c_uint64, I, P]),
        "tb_wcet": (I, [P, ctypes.c_int64, ctypes.c_double, ctypes.c_int64, ctypes.POINTER(ctypes.c_double)]),
        "tb_alpha_star": (I, [P, ctypes.c_int64, ctypes.c_double, ctypes.c_double, ctypes.c_int64,
                              ctypes.c_double, ctypes.c_double, ctypes.c_double,
                              ctypes.POINTER(ctypes.c_double), _I64P]),
        "tb_fit_time_model": (I, [_F64P, _F64P, ctypes.c_int64, ctypes.c_int32, _F64P, _F64P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _LIB = lib
    return lib


# ---------------------------------------------------------------------------
# marshalling helpers
# ---------------------------------------------------------------------------

def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        if not x.is_contiguous():
            raise ValueError("tensor must be contiguous")
        return x.data_ptr()
    raise TypeError("expected a tensor, an integer address or None, got %r" % type(x))


def _nbytes(x) -> int:
    return x.numel() * x.element_size()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        if torch.cuda.is_available():
            return torch.cuda.current_stream().cuda_stream
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(status: int, where: str):
    if status != TB_OK:
        raise TbError(status, where)


class TimeModel(ctypes.Structure):
    """tb_time_model: prefill a N^2 + b N + c and decode step p N_kv + q, seconds."""
    _fields_ = [("a", ctypes.c_double), ("b", ctypes.c_double), ("c", ctypes.c_double),
                ("p", ctypes.c_double), ("q", ctypes.c_double)]


class EvictDesc:
    """tb_evict_desc plus the host arrays it points to (kept alive here)."""

    def __init__(self, *, hq: int, hkv: int, head_dim: int, window: int, pool_k: int,
                 dtype: int, n: Sequence[int], alpha: Sequence[float],
                 kv_offset: Optional[Sequence[int]] = None, kv_rows: Optional[int] = None,
                 out_offset: Optional[Sequence[int]] = None,
                 out_cap: Optional[Sequence[int]] = None, out_rows: Optional[int] = None,
                 flags: int = 0):
        self.n = np.ascontiguousarray(n, dtype=np.int64)
        B = self.n.shape[0]
        self.alpha = np.ascontiguousarray(np.resize(np.asarray(alpha, np.float64), B))
        if kv_offset is None:
            kv_offset = np.concatenate([[0], np.cumsum(self.n)[:-1]]) if B else []
        self.kv_offset = np.ascontiguousarray(kv_offset, dtype=np.int64)
        if kv_rows is None:
            kv_rows = int(self.n.sum())
        if out_cap is None:
            out_cap = [tb_retained_count_ex(int(nb), window, float(a), flags)[1]
                       if nb >= window >= 1 and 0 <= a <= 1 else 0
                       for nb, a in zip(self.n, self.alpha)]
        self.out_cap = np.ascontiguousarray(out_cap, dtype=np.int64)
        if out_offset is None:
            out_offset = np.concatenate([[0], np.cumsum(self.out_cap)[:-1]]) if B else []
        self.out_offset = np.ascontiguousarray(out_offset, dtype=np.int64)
        if out_rows is None:
            out_rows = int((self.out_offset + self.out_cap).max()) if B else 0
        self.hq, self.hkv, self.head_dim, self.window = hq, hkv, head_dim, window
        self.pool_k, self.dtype, self.flags = pool_k, dtype, int(flags)
        self.kv_rows, self.out_rows = int(kv_rows), int(out_rows)
        self.c = _EvictDescC(
            B, hq, hkv, head_dim, window, pool_k, dtype, int(flags),
            self.n.ctypes.data_as(_I64P), self.alpha.ctypes.data_as(_F64P),
            self.kv_offset.ctypes.data_as(_I64P), self.kv_rows,
            self.out_offset.ctypes.data_as(_I64P), self.out_cap.ctypes.data_as(_I64P),
            self.out_rows)

    @property
    def batch(self) -> int:
        return int(self.n.shape[0])

    def ref(self):
        return ctypes.byref(self.c)


class DecodeDesc:
    """tb_decode_desc plus its host arrays."""

    def __init__(self, *, hq: int, hkv: int, head_dim: int, dtype: int, cache_offset,
                 cache_cap, cache_rows: int, max_len: int, out_dtype: int = TB_F32, flags: int = 0,
                 max_ctas: int = 0):
        self.cache_offset = np.ascontiguousarray(cache_offset, dtype=np.int64)
        self.cache_cap = np.ascontiguousarray(cache_cap, dtype=np.int64)
        self.flags = int(flags)
        self.max_ctas = int(max_ctas)
        self.c = _DecodeDescC(
            int(self.cache_offset.shape[0]), hq, hkv, head_dim, dtype, out_dtype,
            self.cache_offset.ctypes.data_as(_I64P), self.cache_cap.ctypes.data_as(_I64P),
            int(cache_rows), int(max_len), self.flags, self.max_ctas)
        self.hq, self.hkv, self.head_dim, self.dtype, self.out_dtype = hq, hkv, head_dim, dtype, out_dtype
        self.cache_rows, self.max_len = int(cache_rows), int(max_len)

    @property
    def batch(self) -> int:
        return int(self.cache_offset.shape[0])

    def ref(self):
        return ctypes.byref(self.c)


# ---------------------------------------------------------------------------
# entry points (same names as the C ABI)
# ---------------------------------------------------------------------------

def tb_status_string(status: int) -> str:
    return load().tb_status_string(status).decode()


def tb_abi_version() -> int:
    return load().tb_abi_version()


def tb_last_error_detail() -> str:
    return load().tb_last_error_detail().decode()


def tb_launch_counter() -> int:
    return int(load().tb_launch_counter())


def tb_retained_count(n: int, window: int, alpha: float):
    k = ctypes.c_int64()
    r = ctypes.c_int64()
    _check(load().tb_retained_count(int(n), int(window), float(alpha), ctypes.byref(k), ctypes.byref(r)),
           "tb_retained_count")
    return k.value, r.value


def tb_retained_count_ex(n: int, window: int, alpha: float, flags: int = 0):
    k = ctypes.c_int64()
    r = ctypes.c_int64()
    _check(load().tb_retained_count_ex(int(n), int(window), float(alpha), int(flags), ctypes.byref(k),
                                       ctypes.byref(r)), "tb_retained_count_ex")
    return k.value, r.value


def tb_evict_layout(desc: EvictDesc):
    s = ctypes.c_int64()
    i = ctypes.c_int64()
    _check(load().tb_evict_layout(desc.ref(), ctypes.byref(s), ctypes.byref(i)), "tb_evict_layout")
    return s.value, i.value


def tb_evict_workspace_size(desc: EvictDesc) -> int:
    b = ctypes.c_size_t()
    _check(load().tb_evict_workspace_size(desc.ref(), ctypes.byref(b)), "tb_evict_workspace_size")
    return b.value


def _ws(workspace, workspace_bytes):
    if workspace_bytes is None:
        workspace_bytes = _nbytes(workspace) if hasattr(workspace, "numel") else 0
    return _ptr(workspace), workspace_bytes


def tb_window_scores(desc: EvictDesc, q_win, K, scores, workspace, workspace_bytes=None, stream=None):
    w, wb = _ws(workspace, workspace_bytes)
    _check(load().tb_window_scores(desc.ref(), _ptr(q_win), _ptr(K), _ptr(scores), w, wb,
                                   _stream(stream)), "tb_window_scores")


def tb_window_scores_lse(desc: EvictDesc, q_win, K, lse, scores, workspace, workspace_bytes=None,
                         stream=None):
    """Window scores from the caller's window-row log-sum-exp (one QK^T pass)."""
    w, wb = _ws(workspace, workspace_bytes)
    _check(load().tb_window_scores_lse(desc.ref(), _ptr(q_win), _ptr(K), _ptr(lse), _ptr(scores), w,
                                       wb, _stream(stream)), "tb_window_scores_lse")


def tb_select_topk(desc: EvictDesc, scores, idx, pooled, workspace, workspace_bytes=None, stream=None):
    w, wb = _ws(workspace, workspace_bytes)
    _check(load().tb_select_topk(desc.ref(), _ptr(scores), _ptr(idx), _ptr(pooled), w, wb,
                                 _stream(stream)), "tb_select_topk")


def tb_select_ctas(desc: EvictDesc) -> int:
    """CTAs (one per SM) the select of this descriptor runs."""
    n = ctypes.c_int32()
    _check(load().tb_select_ctas(desc.ref(), ctypes.byref(n)), "tb_select_ctas")
    return int(n.value)


def tb_gather_kv(desc: EvictDesc, idx, K, V, Kc, Vc, stream=None):
    _check(load().tb_gather_kv(desc.ref(), _ptr(idx), _ptr(K), _ptr(V), _ptr(Kc), _ptr(Vc),
                               _stream(stream)), "tb_gather_kv")


def tb_score_evict(desc: EvictDesc, q_win, K, V, idx, Kc, Vc, pooled, workspace,
                   workspace_bytes=None, stream=None):
    w, wb = _ws(workspace, workspace_bytes)
    _check(load().tb_score_evict(desc.ref(), _ptr(q_win), _ptr(K), _ptr(V), _ptr(idx), _ptr(Kc),
                                 _ptr(Vc), _ptr(pooled), w, wb, _stream(stream)), "tb_score_evict")


def tb_decode_workspace_size(desc: DecodeDesc) -> int:
    b = ctypes.c_size_t()
    _check(load().tb_decode_workspace_size(desc.ref(), ctypes.byref(b)), "tb_decode_workspace_size")
    return b.value


def tb_decode_attn(desc: DecodeDesc, q, Kc, Vc, lens, out, workspace, workspace_bytes=None, stream=None):
    w, wb = _ws(workspace, workspace_bytes)
    _check(load().tb_decode_attn(desc.ref(), _ptr(q), _ptr(Kc), _ptr(Vc), _ptr(lens), _ptr(out), w, wb,
                                 _stream(stream)), "tb_decode_attn")


def tb_decode_workspace_prepare(desc: DecodeDesc, workspace, workspace_bytes=None, stream=None):
    """Zeroes a decode workspace's control words once, for tb_decode_attn_prepared."""
    w, wb = _ws(workspace, workspace_bytes)
    _check(load().tb_decode_workspace_prepare(desc.ref(), w, wb, _stream(stream)),
           "tb_decode_workspace_prepare")


def tb_decode_attn_prepared(desc: DecodeDesc, q, Kc, Vc, lens, out, workspace, workspace_bytes=None,
                            stream=None):
    """tb_decode_attn without the per-call clearing kernel, on a workspace that
    tb_decode_workspace_prepare zeroed once (its status word then stays set
    until the next prepare)."""
    w, wb = _ws(workspace, workspace_bytes)
    _check(load().tb_decode_attn_prepared(desc.ref(), _ptr(q), _ptr(Kc), _ptr(Vc), _ptr(lens), _ptr(out),
                                          w, wb, _stream(stream)), "tb_decode_attn_prepared")


def tb_decode_attn_noalloc(desc: DecodeDesc, q, Kc, Vc, lens, out, stream=None):
    """tb_decode_attn without a workspace, for callers that cannot allocate
    device memory: the library's own 4 MiB device array serves as scratch.
    Calls that overlap on the GPU race on that array."""
    _check(load().tb_decode_attn_noalloc(desc.ref(), _ptr(q), _ptr(Kc), _ptr(Vc), _ptr(lens), _ptr(out),
                                         _stream(stream)), "tb_decode_attn_noalloc")


def tb_decode_noalloc_status(stream=None):
    """(status, raw word) of the array tb_decode_attn_noalloc uses on the
    current device, after waiting for the stream."""
    raw = ctypes.c_int32()
    st = load().tb_decode_noalloc_status(_stream(stream), ctypes.byref(raw))
    if st not in (TB_OK, TB_ERR_TIMEOUT, TB_ERR_INVALID_ARG):
        raise TbError(st, "tb_decode_noalloc_status")
    return st, raw.value


def tb_diag_bounded_wait(workspace, limit_ns: int, arrive: int = 0, workspace_bytes=None, stream=None):
    """Runs the bounded-wait exit on purpose (diagnostic): a wait on a barrier
    that nothing completes gives up after limit_ns; tb_read_status on the
    workspace then reports TB_ERR_TIMEOUT (TB_OK with arrive=1)."""
    w, wb = _ws(workspace, workspace_bytes)
    _check(load().tb_diag_bounded_wait(w, wb, int(limit_ns), int(arrive), _stream(stream)),
           "tb_diag_bounded_wait")


def tb_read_status(workspace, workspace_bytes=None, stream=None):
    """Returns (status, raw status word) after waiting for the stream."""
    w, wb = _ws(workspace, workspace_bytes)
    raw = ctypes.c_int32()
    st = load().tb_read_status(w, wb, _stream(stream), ctypes.byref(raw))
    if st not in (TB_OK, TB_ERR_TIMEOUT, TB_ERR_INVALID_ARG):
        raise TbError(st, "tb_read_status")
    return st, raw.value


def tb_wcet(model: TimeModel, n_x: int, alpha: float, n_w: int) -> float:
    t = ctypes.c_double()
    _check(load().tb_wcet(ctypes.byref(model), int(n_x), float(alpha), int(n_w), ctypes.byref(t)),
           "tb_wcet")
    return t.value


def tb_alpha_star(model: TimeModel, n_x: int, n_hat: float, k: float, n_max: int,
                  t_predict: float, budget: float, alpha_max: float):
    """(alpha*, N_W) of the time budget (host computation)."""
    a = ctypes.c_double()
    n_w = ctypes.c_int64()
    _check(load().tb_alpha_star(ctypes.byref(model), int(n_x), float(n_hat), float(k), int(n_max),
                                float(t_predict), float(budget), float(alpha_max), ctypes.byref(a),
                                ctypes.byref(n_w)), "tb_alpha_star")
    return a.value, n_w.value


def tb_fit_time_model(x, t, degree: int):
    """Least-squares coefficients (highest power first) and MAPE in percent
    of the Eq. 6a (degree 2) or Eq. 6b (degree 1) fit (host computation)."""
    xa = np.ascontiguousarray(x, dtype=np.float64)
    ta = np.ascontiguousarray(t, dtype=np.float64)
    if xa.shape != ta.shape or xa.ndim != 1:
        raise ValueError("x and t must be 1-D and of one length")
    coef = (ctypes.c_double * (max(int(degree), 0) + 1))()
    mape = ctypes.c_double()
    _check(load().tb_fit_time_model(xa.ctypes.data_as(_F64P), ta.ctypes.data_as(_F64P), xa.size,
                                    int(degree), coef, ctypes.byref(mape)), "tb_fit_time_model")
    return list(coef), mape.value
