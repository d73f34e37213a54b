"""Python binding of the C ABI in include/tppsd.h (argument marshalling only).

Every function has the name of the C entry point it calls.  Arrays may be
torch tensors (CUDA or CPU) or numpy arrays; they are passed by pointer.
There is no fallback: if the CUDA library cannot be loaded, every call
raises.
"""
import ctypes as C
import os

import numpy as np

from . import build as _build

TPPSD_OK = 0
TPPSD_ERR_INVALID_ARG = -1
TPPSD_ERR_OOM = -2
TPPSD_ERR_CUDA = -3
TPPSD_ERR_UNSUPPORTED = -4
TPPSD_ERR_ROUND_LIMIT = -5
TPPSD_ERR_TIMEOUT = -6
TPPSD_ERR_NO_DEVICE = -7
TPPSD_WARN_RESAMPLE_CAP = 1
TPPSD_FLAG_NO_BONUS = 1
TPPSD_FLAG_HOST_LOOP = 2
TPPSD_FLAG_PROFILE = 4
TPPSD_FLAG_DEBUG_TRACE = 8
TPPSD_KERNEL_CLASSES = 13


class tppsd_model_cfg(C.Structure):
    _fields_ = [("layers", C.c_int32), ("d_model", C.c_int32), ("heads", C.c_int32),
                ("d_ffn", C.c_int32), ("n_mix", C.c_int32), ("n_marks", C.c_int32),
                ("dtype", C.c_int32), ("encoder", C.c_int32)]


class tppsd_stats(C.Structure):
    _fields_ = [(n, C.c_int64) for n in ("rounds", "drafted", "accepted", "emitted",
                                         "resample_iters", "cap_hits", "loop_iters",
                                         "kernel_launches", "target_keys", "draft_keys",
                                         "prefill_launches")]

    def as_dict(self):
        return {n: int(getattr(self, n)) for n, _ in self._fields_}


class TppsdError(RuntimeError):
    def __init__(self, fn, status, detail=""):
        self.status = status
        super().__init__(f"{fn} failed: {status_str(status)} ({status}) {detail}".strip())


_lib = None
_vp = C.c_void_p


def lib_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Load libtppsd.so (building it first if it is missing or stale)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.build() if build_if_missing else _build.LIB
    if not os.path.exists(path):
        raise RuntimeError(f"CUDA library not built: {path}")
    L = C.CDLL(path)
    L.tppsd_blob_floats.argtypes = [C.POINTER(tppsd_model_cfg)]
    L.tppsd_blob_floats.restype = C.c_size_t
    L.tppsd_create_models.argtypes = [C.POINTER(tppsd_model_cfg), C.POINTER(tppsd_model_cfg),
                                      _vp, C.c_size_t, _vp, C.c_size_t, C.c_int32, C.c_int32,
                                      C.c_int32, C.POINTER(_vp)]
    L.tppsd_prefill.argtypes = [_vp, C.c_int32, _vp, _vp, C.c_int32, _vp]
    L.tppsd_sample.argtypes = [_vp, C.c_int32, C.c_int32, C.c_int32, C.c_uint64, C.c_uint32,
                               _vp, _vp, _vp, _vp]
    L.tppsd_sample_autoregressive.argtypes = [_vp, C.c_int32, C.c_int32, C.c_uint64, C.c_uint32,
                                              _vp, _vp, _vp, _vp]
    L.tppsd_sample_until.argtypes = [_vp, C.c_int32, C.c_double, C.c_int32, C.c_int32, C.c_uint64,
                                     C.c_uint32, _vp, _vp, _vp, _vp, _vp]
    L.tppsd_sample_autoregressive_until.argtypes = [_vp, C.c_int32, C.c_double, C.c_int32, C.c_uint64,
                                                    C.c_uint32, _vp, _vp, _vp, _vp, _vp]
    L.tppsd_sample_poisson.argtypes = [_vp, C.c_int32, C.c_int32, C.c_int32, C.c_double, _vp,
                                       C.c_uint64, C.c_uint32, _vp, _vp, _vp, _vp]
    L.tppsd_sample_poisson_until.argtypes = [_vp, C.c_int32, C.c_double, C.c_int32, C.c_int32,
                                             C.c_double, _vp, C.c_uint64, C.c_uint32, _vp, _vp, _vp,
                                             _vp, _vp]
    L.tppsd_score.argtypes = [_vp, C.c_int32, C.c_int32, C.c_int32, _vp, _vp, _vp, _vp, _vp, _vp]
    L.tppsd_score_until.argtypes = [_vp, C.c_int32, C.c_int32, C.c_int32, _vp, _vp, C.c_double,
                                    _vp, _vp, _vp, _vp, _vp]
    L.tppsd_score_noalloc.argtypes = [_vp, C.c_int32, C.c_int32, C.c_int32, _vp, _vp, _vp, _vp, _vp]
    L.tppsd_score_noalloc.restype = C.c_int
    L.tppsd_get_stats.argtypes = [_vp, C.POINTER(tppsd_stats)]
    L.tppsd_wait.argtypes = [_vp, C.c_int32]
    L.tppsd_set_limits.argtypes = [_vp, C.c_int32, C.c_int32]
    L.tppsd_get_trace.argtypes = [_vp, C.c_int32, C.c_int32, _vp]
    L.tppsd_fit_poisson_draft.argtypes = [C.c_int32, C.c_int32, _vp, _vp, _vp, C.c_int32,
                                          C.POINTER(C.c_double), _vp]
    L.tppsd_kernel_times.argtypes = [_vp, C.POINTER(C.c_double), C.POINTER(C.c_int64)]
    L.tppsd_kernel_times.restype = C.c_int
    L.tppsd_kernel_class_name.argtypes = [C.c_int32]
    L.tppsd_kernel_class_name.restype = C.c_char_p
    L.tppsd_status_str.argtypes = [C.c_int]
    L.tppsd_status_str.restype = C.c_char_p
    L.tppsd_last_error.argtypes = [_vp]
    L.tppsd_last_error.restype = C.c_char_p
    L.tppsd_destroy.argtypes = [_vp]
    L.tppsd_destroy.restype = None
    for f in ("tppsd_create_models", "tppsd_prefill", "tppsd_sample",
              "tppsd_sample_autoregressive", "tppsd_sample_until", "tppsd_sample_autoregressive_until",
              "tppsd_sample_poisson", "tppsd_sample_poisson_until",
              "tppsd_score", "tppsd_score_until", "tppsd_get_stats", "tppsd_wait",
              "tppsd_set_limits", "tppsd_fit_poisson_draft", "tppsd_get_trace"):
        getattr(L, f).restype = C.c_int
    _lib = L
    return L


def status_str(s: int) -> str:
    return load().tppsd_status_str(s).decode()


def _cfg(c):
    if isinstance(c, tppsd_model_cfg):
        return c
    return tppsd_model_cfg(c.layers, c.d_model, c.heads, c.d_ffn, c.n_mix, c.n_marks, c.dtype,
                           getattr(c, "encoder", 0))


def _ptr(a, dtype=None, n=None, name="array"):
    """Pointer of a contiguous torch tensor / numpy array (None -> NULL)."""
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        if not a.flags["C_CONTIGUOUS"]:
            raise ValueError(f"{name} must be C-contiguous")
        if dtype is not None and a.dtype != np.dtype(dtype):
            raise TypeError(f"{name} must be {np.dtype(dtype)}, got {a.dtype}")
        if n is not None and a.size < n:
            raise ValueError(f"{name} holds {a.size} elements, needs {n}")
        return a.ctypes.data
    import torch
    if not isinstance(a, torch.Tensor):
        raise TypeError(f"{name}: expected a torch tensor or numpy array")
    if not a.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None:
        want = {np.float32: torch.float32, np.float64: torch.float64,
                np.int32: torch.int32}[dtype]
        if a.dtype != want:
            raise TypeError(f"{name} must be {want}, got {a.dtype}")
    if n is not None and a.numel() < n:
        raise ValueError(f"{name} holds {a.numel()} elements, needs {n}")
    return a.data_ptr()


def _stream(stream):
    if stream is None:
        try:
            import torch
            if torch.cuda.is_available():
                return torch.cuda.current_stream().cuda_stream
        except Exception:
            pass
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(fn, st, ctx=None):
    if st < 0:
        detail = ""
        if ctx:
            detail = load().tppsd_last_error(ctx).decode()
        raise TppsdError(fn, st, detail)
    return st


def tppsd_blob_floats(cfg) -> int:
    c = _cfg(cfg)
    return int(load().tppsd_blob_floats(C.byref(c)))


def tppsd_create_models(target, draft, target_blob, draft_blob, max_batch, max_positions,
                        max_gamma):
    """Returns an opaque context handle (int)."""
    L = load()
    ct, cd = _cfg(target), _cfg(draft)
    nt, nd = L.tppsd_blob_floats(C.byref(ct)), L.tppsd_blob_floats(C.byref(cd))
    out = _vp()
    st = L.tppsd_create_models(C.byref(ct), C.byref(cd), _ptr(target_blob, np.float32, nt, "target_blob"),
                               nt, _ptr(draft_blob, np.float32, nd, "draft_blob"), nd,
                               max_batch, max_positions, max_gamma, C.byref(out))
    _check("tppsd_create_models", st)
    return out.value


def tppsd_prefill(ctx, batch, hist_tau, hist_marks, hist_len, stream=None):
    n = batch * hist_len
    st = load().tppsd_prefill(ctx, batch, _ptr(hist_tau, np.float32, n, "hist_tau"),
                              _ptr(hist_marks, np.int32, n, "hist_marks"), hist_len, _stream(stream))
    return _check("tppsd_prefill", st, ctx)


def tppsd_sample(ctx, batch, n_events, gamma, seed, flags, out_tau, out_t, out_marks, stream=None):
    n = batch * n_events
    st = load().tppsd_sample(ctx, batch, n_events, gamma, seed, flags,
                             _ptr(out_tau, np.float32, n, "out_tau"),
                             _ptr(out_t, np.float64, n, "out_t"),
                             _ptr(out_marks, np.int32, n, "out_marks"), _stream(stream))
    return _check("tppsd_sample", st, ctx)


def tppsd_sample_autoregressive(ctx, batch, n_events, seed, flags, out_tau, out_t, out_marks,
                                stream=None):
    n = batch * n_events
    st = load().tppsd_sample_autoregressive(ctx, batch, n_events, seed, flags,
                                            _ptr(out_tau, np.float32, n, "out_tau"),
                                            _ptr(out_t, np.float64, n, "out_t"),
                                            _ptr(out_marks, np.int32, n, "out_marks"),
                                            _stream(stream))
    return _check("tppsd_sample_autoregressive", st, ctx)


def tppsd_sample_until(ctx, batch, t_end, max_events, gamma, seed, flags, out_tau, out_t, out_marks,
                       out_count, stream=None):
    n = batch * max_events
    st = load().tppsd_sample_until(ctx, batch, float(t_end), max_events, gamma, seed, flags,
                                   _ptr(out_tau, np.float32, n, "out_tau"),
                                   _ptr(out_t, np.float64, n, "out_t"),
                                   _ptr(out_marks, np.int32, n, "out_marks"),
                                   _ptr(out_count, np.int32, batch, "out_count"), _stream(stream))
    return _check("tppsd_sample_until", st, ctx)


def tppsd_sample_autoregressive_until(ctx, batch, t_end, max_events, seed, flags, out_tau, out_t,
                                      out_marks, out_count, stream=None):
    n = batch * max_events
    st = load().tppsd_sample_autoregressive_until(ctx, batch, float(t_end), max_events, seed, flags,
                                                  _ptr(out_tau, np.float32, n, "out_tau"),
                                                  _ptr(out_t, np.float64, n, "out_t"),
                                                  _ptr(out_marks, np.int32, n, "out_marks"),
                                                  _ptr(out_count, np.int32, batch, "out_count"),
                                                  _stream(stream))
    return _check("tppsd_sample_autoregressive_until", st, ctx)


def _host_f64(a, name):
    a = np.ascontiguousarray(np.asarray(a, dtype=np.float64))
    if a.ndim != 1:
        raise ValueError(f"{name}: expected a 1-D host array")
    return a, a.ctypes.data_as(_vp)


def tppsd_sample_poisson(ctx, batch, n_events, gamma, rate, mark_probs, seed, flags, out_tau, out_t,
                         out_marks, stream=None):
    n = batch * n_events
    probs, pp = _host_f64(mark_probs, "mark_probs")
    st = load().tppsd_sample_poisson(ctx, batch, n_events, gamma, float(rate), pp, seed, flags,
                                     _ptr(out_tau, np.float32, n, "out_tau"),
                                     _ptr(out_t, np.float64, n, "out_t"),
                                     _ptr(out_marks, np.int32, n, "out_marks"), _stream(stream))
    del probs
    return _check("tppsd_sample_poisson", st, ctx)


def tppsd_sample_poisson_until(ctx, batch, t_end, max_events, gamma, rate, mark_probs, seed, flags,
                               out_tau, out_t, out_marks, out_count, stream=None):
    n = batch * max_events
    probs, pp = _host_f64(mark_probs, "mark_probs")
    st = load().tppsd_sample_poisson_until(ctx, batch, float(t_end), max_events, gamma, float(rate),
                                           pp, seed, flags,
                                           _ptr(out_tau, np.float32, n, "out_tau"),
                                           _ptr(out_t, np.float64, n, "out_t"),
                                           _ptr(out_marks, np.int32, n, "out_marks"),
                                           _ptr(out_count, np.int32, batch, "out_count"),
                                           _stream(stream))
    del probs
    return _check("tppsd_sample_poisson_until", st, ctx)


def tppsd_fit_poisson_draft(tau, marks, n_marks, t_window=None):
    """(rate, mark_probs) of the App. D.3 Poisson draft fitted by maximum
    likelihood on tau / marks [batch][len]; t_window [batch] optional."""
    if isinstance(tau, np.ndarray):
        tau = np.ascontiguousarray(tau, np.float32)
        marks = np.ascontiguousarray(marks, np.int32)
    B, n = tau.shape
    win = None
    if t_window is not None:
        win, _ = _host_f64(t_window, "t_window")
        if win.size != B:
            raise ValueError("t_window must hold one value per sequence")
    rate = C.c_double()
    probs = np.zeros(n_marks, np.float64)
    st = load().tppsd_fit_poisson_draft(B, n, _ptr(tau, np.float32, B * n, "tau"),
                                        _ptr(marks, np.int32, B * n, "marks"),
                                        None if win is None else win.ctypes.data, n_marks,
                                        C.byref(rate), probs.ctypes.data)
    _check("tppsd_fit_poisson_draft", st)
    return rate.value, probs


def tppsd_score_until(ctx, which, batch, length, tau, marks, t_end, out_heads, out_logg, out_logf,
                      out_logS, stream=None):
    n = batch * length
    st = load().tppsd_score_until(ctx, which, batch, length, _ptr(tau, np.float32, n, "tau"),
                                  _ptr(marks, np.int32, n, "marks"), float(t_end),
                                  _ptr(out_heads, np.float32, None, "out_heads"),
                                  _ptr(out_logg, np.float32, n, "out_logg"),
                                  _ptr(out_logf, np.float32, n, "out_logf"),
                                  _ptr(out_logS, np.float64, batch, "out_logS"), _stream(stream))
    return _check("tppsd_score_until", st, ctx)


def tppsd_score(ctx, which, batch, length, tau, marks, out_heads, out_logg, out_logf, stream=None):
    n = batch * length
    st = load().tppsd_score(ctx, which, batch, length, _ptr(tau, np.float32, n, "tau"),
                            _ptr(marks, np.int32, n, "marks"), _ptr(out_heads, np.float32, None, "out_heads"),
                            _ptr(out_logg, np.float32, n, "out_logg"),
                            _ptr(out_logf, np.float32, n, "out_logf"), _stream(stream))
    return _check("tppsd_score", st, ctx)


def tppsd_score_noalloc(ctx, which, batch, length, tau, marks, out_logg, out_logf, stream=None):
    """Scoring whose working memory is a fixed device array of the library:
    the call allocates nothing.  All arrays must be CUDA tensors."""
    n = batch * length
    st = load().tppsd_score_noalloc(ctx, which, batch, length, _ptr(tau, np.float32, n, "tau"),
                                    _ptr(marks, np.int32, n, "marks"),
                                    _ptr(out_logg, np.float32, n, "out_logg"),
                                    _ptr(out_logf, np.float32, n, "out_logf"), _stream(stream))
    return _check("tppsd_score_noalloc", st, ctx)


def tppsd_get_stats(ctx):
    """(status, stats dict) of the last sampling call; synchronises."""
    s = tppsd_stats()
    st = load().tppsd_get_stats(ctx, C.byref(s))
    _check("tppsd_get_stats", st, ctx)
    return st, s.as_dict()


def tppsd_kernel_times(ctx):
    """{class name: (total ms, launches)} of the last profiled call."""
    L = load()
    ms = (C.c_double * TPPSD_KERNEL_CLASSES)()
    n = (C.c_int64 * TPPSD_KERNEL_CLASSES)()
    _check("tppsd_kernel_times", L.tppsd_kernel_times(ctx, ms, n), ctx)
    return {L.tppsd_kernel_class_name(i).decode(): (ms[i], int(n[i]))
            for i in range(TPPSD_KERNEL_CLASSES)}


def tppsd_kernel_class_name(cls):
    return load().tppsd_kernel_class_name(cls).decode()


def tppsd_get_trace(ctx, batch, n_events, out=None):
    """[batch][n_events][4] decision records of the last traced sampling call
    (a new float32 numpy array unless `out` is given)."""
    if out is None:
        out = np.zeros((batch, n_events, 4), np.float32)
    st = load().tppsd_get_trace(ctx, batch, n_events, _ptr(out, np.float32, batch * n_events * 4, "out"))
    _check("tppsd_get_trace", st, ctx)
    return out


def tppsd_set_limits(ctx, resample_cap, max_rounds):
    return _check("tppsd_set_limits", load().tppsd_set_limits(ctx, resample_cap, max_rounds), ctx)


def tppsd_wait(ctx, timeout_ms):
    return load().tppsd_wait(ctx, timeout_ms)


def tppsd_status_str(status):
    return status_str(status)


def tppsd_last_error(ctx):
    return load().tppsd_last_error(ctx).decode()


def tppsd_destroy(ctx):
    if ctx:
        load().tppsd_destroy(ctx)
