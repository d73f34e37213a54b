"""ctypes front of the C oracle (oracle/tppsd_oracle.c) -- test infrastructure.

Argument marshalling only; every computation happens in the C file.
"""
import ctypes as C
import os

import numpy as np

from . import build as _build

FLAG_NO_BONUS = 1
_lib = None

_i32p = np.ctypeslib.ndpointer(np.int32, flags="C_CONTIGUOUS")
_f32p = np.ctypeslib.ndpointer(np.float32, flags="C_CONTIGUOUS")
_f64p = np.ctypeslib.ndpointer(np.float64, flags="C_CONTIGUOUS")
_i64p = np.ctypeslib.ndpointer(np.int64, flags="C_CONTIGUOUS")
_u32p = np.ctypeslib.ndpointer(np.uint32, flags="C_CONTIGUOUS")


def _opt(p):
    """ndpointer that also accepts None."""
    class _P(p):
        @classmethod
        def from_param(cls, obj):
            if obj is None:
                return None
            return p.from_param(obj)
    return _P


def lib():
    global _lib
    if _lib is None:
        path = _build.build()
        L = C.CDLL(path)
        L.oracle_philox4x32.argtypes = [_u32p, _u32p, _u32p]
        L.oracle_uniforms.argtypes = [C.c_uint64, C.c_uint32, C.c_uint32, C.c_uint32, _f64p]
        L.oracle_round_bf16.argtypes = [C.c_double]
        L.oracle_round_bf16.restype = C.c_double
        L.oracle_temporal_encoding.argtypes = [C.c_int32, C.c_double, _f64p]
        L.oracle_score.argtypes = [_i32p, _f32p, C.c_int64, C.c_int32, C.c_int32, _f32p, _i32p,
                                   _opt(_f64p), _opt(_f64p), _opt(_f64p), C.c_int32, C.c_int32]
        L.oracle_sample_ar.argtypes = [_i32p, _f32p, C.c_int64, C.c_int32, C.c_int32, _f32p, _i32p,
                                       C.c_int32, C.c_uint64, C.c_int32, _opt(_i32p),
                                       _f64p, _f64p, _i32p, _f64p, C.c_int32]
        L.oracle_sample_sd.argtypes = [_i32p, _f32p, C.c_int64, _i32p, _f32p, C.c_int64,
                                       C.c_int32, C.c_int32, _f32p, _i32p, C.c_int32, C.c_int32,
                                       C.c_uint64, C.c_uint32, C.c_int32, _opt(_i32p),
                                       _f64p, _f64p, _i32p, _f64p, _i64p, C.c_int32]
        L.oracle_log_g.argtypes = [C.c_int32, _f64p, C.c_double]
        L.oracle_log_g.restype = C.c_double
        L.oracle_log_f.argtypes = [C.c_int32, _f64p, C.c_int32]
        L.oracle_log_f.restype = C.c_double
        L.oracle_sample_head.argtypes = [C.c_int32, C.c_int32, _f64p, C.c_int32, C.c_uint64,
                                         _f64p, _opt(_i32p)]
        L.oracle_resample_time.argtypes = [C.c_int32, _f64p, _f64p, C.c_int32, C.c_uint64,
                                           _f64p, _opt(_i32p)]
        L.oracle_resample_mark.argtypes = [C.c_int32, C.c_int32, _f64p, _f64p, C.c_int32,
                                           C.c_uint64, _i32p]
        L.oracle_toy_sd.argtypes = [C.c_int32, C.c_int32, _f64p, _f64p, C.c_int32, C.c_int32,
                                    C.c_int32, C.c_uint64, C.c_uint32, _f64p, _i32p, _i64p]
        L.oracle_toy_ar.argtypes = [C.c_int32, C.c_int32, _f64p, C.c_int32, C.c_int32,
                                    C.c_uint64, _f64p, _i32p]
        L.oracle_sample_ar_until.argtypes = [_i32p, _f32p, C.c_int64, C.c_int32, C.c_int32, _f32p,
                                             _i32p, C.c_int32, C.c_double, C.c_uint64, C.c_int32,
                                             _opt(_i32p), _f64p, _f64p, _i32p, _f64p, _i32p, C.c_int32]
        L.oracle_sample_sd_until.argtypes = [_i32p, _f32p, C.c_int64, _i32p, _f32p, C.c_int64,
                                             C.c_int32, C.c_int32, _f32p, _i32p, C.c_int32, C.c_double,
                                             C.c_int32, C.c_uint64, C.c_uint32, C.c_int32, _opt(_i32p),
                                             _f64p, _f64p, _i32p, _f64p, _i32p, _i64p, C.c_int32]
        L.oracle_score_survival.argtypes = [_i32p, _f32p, C.c_int64, C.c_int32, C.c_int32, _f32p,
                                            _i32p, C.c_double, _f64p, C.c_int32, C.c_int32]
        L.oracle_model_temporal_encoding.argtypes = [_i32p, _f32p, C.c_int64, C.c_double, _f64p]
        L.oracle_model_temporal_encoding.restype = C.c_int
        L.oracle_log_survival.argtypes = [C.c_int32, _f64p, C.c_double]
        L.oracle_log_survival.restype = C.c_double
        L.oracle_sample_sd_poisson_until.argtypes = [
            _i32p, _f32p, C.c_int64, C.c_int32, C.c_int32, _f32p, _i32p, C.c_int32, C.c_double,
            C.c_int32, C.c_double, _f64p, C.c_uint64, C.c_uint32, C.c_int32, _opt(_i32p),
            _f64p, _f64p, _i32p, _f64p, _i32p, _i64p, C.c_int32]
        L.oracle_sample_poisson.argtypes = [C.c_double, C.c_int32, _f64p, C.c_int32, C.c_uint64,
                                            _f64p, _i32p]
        L.oracle_resample_time_poisson.argtypes = [C.c_int32, _f64p, C.c_double, C.c_int32,
                                                   C.c_uint64, _f64p, _i32p]
        L.oracle_toy_sd_poisson.argtypes = [C.c_int32, C.c_int32, _f64p, C.c_double, _f64p,
                                            C.c_int32, C.c_int32, C.c_int32, C.c_uint64, C.c_uint32,
                                            _f64p, _i32p, _i64p]
        for f in ("oracle_score", "oracle_sample_ar", "oracle_sample_sd", "oracle_toy_sd",
                  "oracle_toy_ar", "oracle_sample_ar_until", "oracle_sample_sd_until",
                  "oracle_score_survival", "oracle_sample_sd_poisson_until", "oracle_sample_poisson",
                  "oracle_resample_time_poisson", "oracle_toy_sd_poisson"):
            getattr(L, f).restype = C.c_int
        _lib = L
    return _lib


def _cfg(cfg):
    return np.array([cfg.layers, cfg.d_model, cfg.heads, cfg.d_ffn, cfg.n_mix, cfg.n_marks,
                     cfg.dtype, getattr(cfg, "encoder", 0)], np.int32)


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def _check(rc, what):
    if rc != 0:
        raise ValueError(f"{what} rejected its arguments (rc={rc})")


def philox4x32(ctr, key):
    out = np.zeros(4, np.uint32)
    lib().oracle_philox4x32(_c(ctr, np.uint32), _c(key, np.uint32), out)
    return out


def uniforms(seed, seq, pos, block):
    u = np.zeros(4)
    lib().oracle_uniforms(seed, seq, pos, block, u)
    return u


def round_bf16(x: float) -> float:
    return lib().oracle_round_bf16(float(x))


def temporal_encoding(d: int, t: float):
    out = np.zeros(d)
    lib().oracle_temporal_encoding(d, float(t), out)
    return out


def head_width(cfg):
    return 3 * cfg.n_mix + cfg.n_marks


def score(cfg, blob, tau, marks, recompute=False, nthreads=0, heads=True):
    """Teacher-forced heads and per-event log g / log f of one model."""
    tau = _c(tau, np.float32)
    marks = _c(marks, np.int32)
    B, n = tau.shape
    hd = np.full((B, n, head_width(cfg)), np.nan) if heads else None
    lg = np.zeros((B, n))
    lf = np.zeros((B, n))
    _check(lib().oracle_score(_cfg(cfg), _c(blob, np.float32), blob.size, B, n, tau, marks,
                              hd, lg, lf, int(recompute), nthreads), "oracle_score")
    return hd, lg, lf


def _ids(seq_ids, B):
    if seq_ids is None:
        return None
    ids = np.ascontiguousarray(seq_ids, np.int32)
    if ids.shape != (B,):
        raise ValueError("seq_ids must have one entry per sequence")
    return ids


def sample_ar(cfg_t, blob_t, hist_tau, hist_marks, n_events, seed, recompute=False, nthreads=0,
              seq_ids=None):
    hist_tau = _c(hist_tau, np.float32)
    hist_marks = _c(hist_marks, np.int32)
    B, H = hist_tau.shape
    tau = np.zeros((B, n_events)); t = np.zeros((B, n_events))
    k = np.zeros((B, n_events), np.int32); mg = np.zeros((B, n_events))
    _check(lib().oracle_sample_ar(_cfg(cfg_t), _c(blob_t, np.float32), blob_t.size, B, H,
                                  hist_tau, hist_marks, n_events, seed, int(recompute),
                                  _ids(seq_ids, B), tau, t, k, mg, nthreads), "oracle_sample_ar")
    return dict(tau=tau, t=t, k=k, margin=mg)


def sample_sd(cfg_t, blob_t, cfg_d, blob_d, hist_tau, hist_marks, n_events, gamma, seed,
              flags=0, recompute=False, nthreads=0, seq_ids=None):
    hist_tau = _c(hist_tau, np.float32)
    hist_marks = _c(hist_marks, np.int32)
    B, H = hist_tau.shape
    tau = np.zeros((B, n_events)); t = np.zeros((B, n_events))
    k = np.zeros((B, n_events), np.int32); mg = np.zeros((B, n_events))
    st = np.zeros((B, 5), np.int64)
    _check(lib().oracle_sample_sd(_cfg(cfg_t), _c(blob_t, np.float32), blob_t.size,
                                  _cfg(cfg_d), _c(blob_d, np.float32), blob_d.size, B, H,
                                  hist_tau, hist_marks, n_events, gamma, seed, flags,
                                  int(recompute), _ids(seq_ids, B), tau, t, k, mg, st, nthreads),
           "oracle_sample_sd")
    return dict(tau=tau, t=t, k=k, margin=mg, stats=st)


def sample_ar_until(cfg_t, blob_t, hist_tau, hist_marks, max_events, t_end, seed, recompute=False,
                    nthreads=0, seq_ids=None):
    """AR sampling until the end time t_end (Alg. 1's stop rule) or
    max_events; count[b] events with t <= t_end fill the first slots."""
    hist_tau = _c(hist_tau, np.float32)
    hist_marks = _c(hist_marks, np.int32)
    B, H = hist_tau.shape
    N = max_events
    tau = np.zeros((B, N)); t = np.zeros((B, N))
    k = np.zeros((B, N), np.int32); mg = np.zeros((B, N)); cnt = np.zeros(B, np.int32)
    _check(lib().oracle_sample_ar_until(_cfg(cfg_t), _c(blob_t, np.float32), blob_t.size, B, H,
                                        hist_tau, hist_marks, N, float(t_end), seed, int(recompute),
                                        _ids(seq_ids, B), tau, t, k, mg, cnt, nthreads),
           "oracle_sample_ar_until")
    return dict(tau=tau, t=t, k=k, margin=mg, count=cnt)


def sample_sd_until(cfg_t, blob_t, cfg_d, blob_d, hist_tau, hist_marks, max_events, t_end, gamma,
                    seed, flags=0, recompute=False, nthreads=0, seq_ids=None):
    """TPP-SD until the end time t_end (Alg. 1's stop rule) or max_events."""
    hist_tau = _c(hist_tau, np.float32)
    hist_marks = _c(hist_marks, np.int32)
    B, H = hist_tau.shape
    N = max_events
    tau = np.zeros((B, N)); t = np.zeros((B, N))
    k = np.zeros((B, N), np.int32); mg = np.zeros((B, N)); cnt = np.zeros(B, np.int32)
    st = np.zeros((B, 5), np.int64)
    _check(lib().oracle_sample_sd_until(_cfg(cfg_t), _c(blob_t, np.float32), blob_t.size,
                                        _cfg(cfg_d), _c(blob_d, np.float32), blob_d.size, B, H,
                                        hist_tau, hist_marks, N, float(t_end), gamma, seed, flags,
                                        int(recompute), _ids(seq_ids, B), tau, t, k, mg, cnt, st,
                                        nthreads), "oracle_sample_sd_until")
    return dict(tau=tau, t=t, k=k, margin=mg, count=cnt, stats=st)


def score_survival(cfg, blob, tau, marks, t_end, recompute=False, nthreads=0):
    """log S(t_end - t_last) per sequence (survival term of Eq. 2)."""
    tau = _c(tau, np.float32)
    marks = _c(marks, np.int32)
    B, n = tau.shape
    out = np.zeros(B)
    _check(lib().oracle_score_survival(_cfg(cfg), _c(blob, np.float32), blob.size, B, n, tau, marks,
                                       float(t_end), out, int(recompute), nthreads),
           "oracle_score_survival")
    return out


def log_survival(M, head, u):
    """log(1 - G(u)) of one head's log-normal mixture."""
    return lib().oracle_log_survival(M, _c(head, np.float64), float(u))


def model_temporal_encoding(cfg, blob, t):
    """z(t) of a model's encoder (THP, SAHP or AttNHP form)."""
    out = np.zeros(cfg.d_model)
    _check(lib().oracle_model_temporal_encoding(_cfg(cfg), _c(blob, np.float32), blob.size, float(t), out),
           "oracle_model_temporal_encoding")
    return out


def log_g(M, head, tau):
    head = _c(head, np.float64)
    return np.array([lib().oracle_log_g(M, head, float(x)) for x in np.atleast_1d(tau)])


def sample_head(M, K, head, n, seed):
    tau = np.zeros(n); k = np.zeros(n, np.int32)
    lib().oracle_sample_head(M, K, _c(head, np.float64), n, seed, tau, k)
    return tau, k


def resample_time(M, head_t, head_d, n, seed):
    tau = np.zeros(n); it = np.zeros(n, np.int32)
    lib().oracle_resample_time(M, _c(head_t, np.float64), _c(head_d, np.float64), n, seed, tau, it)
    return tau, it


def resample_mark(M, K, head_t, head_d, n, seed):
    k = np.zeros(n, np.int32)
    lib().oracle_resample_mark(M, K, _c(head_t, np.float64), _c(head_d, np.float64), n, seed, k)
    return k


def toy_sd(M, K, table_t, table_d, B, N, gamma, seed, flags=0):
    tau = np.zeros((B, N)); k = np.zeros((B, N), np.int32); st = np.zeros((B, 5), np.int64)
    _check(lib().oracle_toy_sd(M, K, _c(table_t, np.float64), _c(table_d, np.float64), B, N,
                               gamma, seed, flags, tau, k, st), "oracle_toy_sd")
    return tau, k, st


def sample_sd_poisson_until(cfg_t, blob_t, hist_tau, hist_marks, max_events, t_end, gamma, lam,
                            p_marks, seed, flags=0, recompute=False, nthreads=0, seq_ids=None):
    """TPP-SD with the Poisson draft of App. D.3 (rate lam, mark
    probabilities p_marks) until t_end or max_events."""
    hist_tau = _c(hist_tau, np.float32)
    hist_marks = _c(hist_marks, np.int32)
    B, H = hist_tau.shape
    N = max_events
    tau = np.zeros((B, N)); t = np.zeros((B, N))
    k = np.zeros((B, N), np.int32); mg = np.zeros((B, N)); cnt = np.zeros(B, np.int32)
    st = np.zeros((B, 5), np.int64)
    _check(lib().oracle_sample_sd_poisson_until(
        _cfg(cfg_t), _c(blob_t, np.float32), blob_t.size, B, H, hist_tau, hist_marks, N,
        float(t_end), gamma, float(lam), _c(p_marks, np.float64), seed, flags, int(recompute),
        _ids(seq_ids, B), tau, t, k, mg, cnt, st, nthreads), "oracle_sample_sd_poisson_until")
    return dict(tau=tau, t=t, k=k, margin=mg, count=cnt, stats=st)


def sample_sd_poisson(cfg_t, blob_t, hist_tau, hist_marks, n_events, gamma, lam, p_marks, seed,
                      **kw):
    """Fixed-count form (t_end = +inf)."""
    return sample_sd_poisson_until(cfg_t, blob_t, hist_tau, hist_marks, n_events, np.inf, gamma,
                                   lam, p_marks, seed, **kw)


def sample_poisson(lam, p, n, seed):
    tau = np.zeros(n); k = np.zeros(n, np.int32)
    p = _c(p, np.float64)
    _check(lib().oracle_sample_poisson(float(lam), p.size, p, n, seed, tau, k), "oracle_sample_poisson")
    return tau, k


def resample_time_poisson(M, head_t, lam, n, seed):
    tau = np.zeros(n); it = np.zeros(n, np.int32)
    _check(lib().oracle_resample_time_poisson(M, _c(head_t, np.float64), float(lam), n, seed, tau, it),
           "oracle_resample_time_poisson")
    return tau, it


def toy_sd_poisson(M, K, table_t, lam, p, B, N, gamma, seed, flags=0):
    tau = np.zeros((B, N)); k = np.zeros((B, N), np.int32); st = np.zeros((B, 5), np.int64)
    _check(lib().oracle_toy_sd_poisson(M, K, _c(table_t, np.float64), float(lam), _c(p, np.float64),
                                       B, N, gamma, seed, flags, tau, k, st), "oracle_toy_sd_poisson")
    return tau, k, st


def toy_ar(M, K, table_t, B, N, seed):
    tau = np.zeros((B, N)); k = np.zeros((B, N), np.int32)
    _check(lib().oracle_toy_ar(M, K, _c(table_t, np.float64), B, N, seed, tau, k),
           "oracle_toy_ar")
    return tau, k


def cores() -> int:
    return os.cpu_count() or 1
