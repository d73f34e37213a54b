"""Helpers of the GPU parity tests: build a sampler, compare with the oracle."""
import numpy as np

from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN

# Tolerances (stated by the method's accuracy target): per-position log
# densities 1e-4 absolute in fp32, 5e-3 with bf16 weights; fp32 sequences
# identical except after a decision whose margin is below 1e-6.
TOL_FP32 = 1e-4
TOL_BF16 = 5e-3
MARGIN_FP32 = 1e-6
# bf16 sequences: GPU and oracle differ in the last bf16 bit of an
# activation now and then, which moves a log density by up to the bf16
# tolerance.  A test u < exp(log g_T - log g_D) compares u with a ratio that
# both log densities move: with each within TOL_BF16 the ratio moves by at
# most exp(2 TOL_BF16) - 1 ~ 1e-2, and a categorical draw's cumulative
# probabilities by less.  So a divergence is excused only after an oracle
# decision closer than that to its threshold.
MARGIN_BF16 = 1e-2
# sampled bf16 times are compared to this relative tolerance (a time is
# exp(mu + sigma eps) with mu, sigma within TOL_BF16; several events add)
RTOL_BF16 = 2e-2
# bf16 sampling tests on models with the workloads' weight scale: at least
# this fraction of sequences must match the oracle event for event, and at
# most one sequence of a small batch may diverge (only ever after a decision
# within MARGIN_BF16 of its threshold)
MIN_IDENTICAL_FRAC = 0.9


def min_identical(B):
    """Sequences of a batch of B that must match the oracle exactly."""
    return min(B - 1, int(np.ceil(MIN_IDENTICAL_FRAC * B))) if B > 1 else 1


def make_sampler(tcfg, dcfg, bt, bd, B, n_max, gmax):
    from paper_2507_09252_gb300.sampler import Sampler
    return Sampler(tcfg, dcfg, bt, bd, max_batch=B, max_positions=n_max, max_gamma=gmax)


def to_np(out):
    return {k: v.detach().cpu().numpy() for k, v in out.items()}


def first_divergence(g, o, rtol=1e-4):
    """Index of the first event where GPU and oracle differ (mark differs or
    tau differs beyond rtol), -1 if none."""
    bad = (g["k"] != o["k"]) | (np.abs(g["tau"] - o["tau"]) > rtol * np.maximum(np.abs(o["tau"]), 1e-6))
    idx = np.argmax(bad)
    return int(idx) if bad[idx] else -1


def compare_sequences(gpu, ora, margin_tol, rtol=1e-4, gpu_trace=None):
    """Per sequence: identical, or first divergence preceded (at or before)
    by an oracle decision margin < margin_tol.  With gpu_trace (the
    [B][N][4] records of a TPPSD_FLAG_DEBUG_TRACE call) the GPU's own test
    margins count too.  Returns (identical, excused, failures[list of
    (b, idx, min_margin)])."""
    B = gpu["k"].shape[0]
    ident, excused, fails = 0, 0, []
    for b in range(B):
        g = {k: gpu[k][b] for k in ("tau", "k")}
        o = {k: ora[k][b] for k in ("tau", "k")}
        i = first_divergence(g, o, rtol)
        if i < 0:
            ident += 1
            continue
        mm = float(np.min(ora["margin"][b, :i + 1]))
        if gpu_trace is not None:
            gm = np.abs(gpu_trace[b, :i + 1, :2])
            if np.isfinite(gm).any():
                mm = min(mm, float(np.nanmin(gm)))
        if mm < margin_tol:
            excused += 1
        else:
            fails.append((b, i, mm))
    return ident, excused, fails


SMALL_T = CF.ModelCfg(2, 32, 2, 64, 4, 3, CF.FP32)
SMALL_D = CF.ModelCfg(1, 16, 1, 32, 4, 3, CF.FP32)


def small_models(gain=6.0, shift=True, dtype=CF.FP32, tcfg=None, dcfg=None, seed=11):
    tcfg = tcfg or CF.ModelCfg(**{**SMALL_T.__dict__, "dtype": dtype})
    dcfg = dcfg or CF.ModelCfg(**{**SMALL_D.__dict__, "dtype": dtype})
    bt = IN.model_blob(tcfg, seed, 0, head_gain=gain)
    bd = IN.model_blob(dcfg, seed, 1, head_gain=gain)
    if shift:
        K = dcfg.n_marks
        bd = IN.shift_blob(dcfg, bd, **{"head.b_mu": 0.4, "head.b_s": -0.2,
                                        "head.b_k2": np.linspace(0.5, -0.5, K)})
    return tcfg, dcfg, bt, bd


def hist(B, H, K, seed=0):
    rng = np.random.default_rng(seed)
    return (rng.exponential(1.0, (B, H)).astype(np.float32),
            rng.integers(0, K, (B, H)).astype(np.int32))
