"""The oracle's TPP-SD output law equals autoregressive target sampling.

App. A.2 proves that accept/reject plus the adjusted distributions (Eq. 3-4,
Theorem 1) reproduce g_T and f_T; the paper's experiments check SD against AR
with KS tests (Sec. 5.1, App. A.4).  These tests check the oracle against
exact laws where one exists (toy Markov models) and against AR and the
target's own conditional densities otherwise, with >= 1e5 events.
"""
import numpy as np
import pytest
from scipy import stats

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from tests import helpers as HP

P_MIN = 1e-3


def _toy_tables(rng, M, K, spread=1.0):
    return np.stack([HP.random_head(rng, M, K, mu_scale=spread, k_scale=spread) for _ in range(K)])


def _markov_law(table, M, K, n):
    """Exact law of the first n marks: a Markov chain from mark 0 with
    transition f_T(. | previous mark)."""
    f = np.exp(table[:, 3 * M:])
    law = {(): 1.0}
    for _ in range(n):
        law = {seq + (k,): p * f[seq[-1] if seq else 0, k] for seq, p in law.items() for k in range(K)}
    return law


@pytest.mark.parametrize("gamma,flags", [(1, 0), (2, 0), (3, 0), (3, O.FLAG_NO_BONUS)])
def test_toy_sd_matches_exact_markov_law(gamma, flags):
    """Brute force on a toy with K=3: the law of (k1,k2,k3) under SD equals
    the product of f_T transitions enumerated exactly; times pass a PIT test
    against g_T(. | previous mark); tau and k are independent given the
    past; and the draft differs enough that rejections (both kinds) occur."""
    rng = np.random.default_rng(42)
    M, K, N, B = 3, 3, 3, 100000
    tT = _toy_tables(rng, M, K)
    tD = _toy_tables(rng, M, K)
    tau, k, st = O.toy_sd(M, K, tT, tD, B, N, gamma, seed=17, flags=flags)
    law = _markov_law(tT, M, K, N)
    keys = sorted(law)
    idx = {key: i for i, key in enumerate(keys)}
    counts = np.bincount([idx[tuple(r)] for r in k], minlength=len(keys))
    assert HP.chi2_pvalue(counts, B * np.array([law[key] for key in keys])) > P_MIN
    prev = np.concatenate([np.zeros((B, 1), np.int32), k[:, :-1]], 1)
    u = np.empty_like(tau)
    for j in range(K):
        sel = prev == j
        u[sel] = HP.mixture_cdf(tT[j], M, tau[sel])
    assert stats.kstest(u.ravel(), "uniform").pvalue > P_MIN
    # independence of the time quantile and the mark, given previous mark 0
    sel = prev[:, 0] == 0
    table = np.histogram2d(np.minimum((u[sel, 0] * 4).astype(int), 3), k[sel, 0],
                           bins=[4, K], range=[[0, 4], [0, K]])[0]
    assert stats.chi2_contingency(table)[1] > P_MIN
    acc = st[:, 2].sum() / st[:, 1].sum()
    assert 0.05 < acc < 0.95
    assert st[:, 3].sum() > 0            # Theorem 1 loop ran


def test_toy_sd_identical_draft_equals_ar():
    """draft == target: every ratio is 1, nothing is rejected, and SD
    reproduces AR event for event (same slot per position)."""
    rng = np.random.default_rng(1)
    M, K = 2, 4
    tT = _toy_tables(rng, M, K)
    a_tau, a_k = O.toy_ar(M, K, tT, 50, 30, seed=5)
    s_tau, s_k, st = O.toy_sd(M, K, tT, tT, 50, 30, 4, seed=5)
    assert np.array_equal(a_k, s_k) and np.array_equal(a_tau, s_tau)
    assert st[:, 1].sum() == st[:, 2].sum()


def test_toy_no_bonus_is_gamma_invariant():
    """Without the bonus event every position p is decided by its own slots
    from the same prefix, so the output does not depend on gamma."""
    rng = np.random.default_rng(2)
    M, K = 2, 3
    tT, tD = _toy_tables(rng, M, K), _toy_tables(rng, M, K)
    ref = O.toy_sd(M, K, tT, tD, 200, 25, 1, seed=8, flags=O.FLAG_NO_BONUS)
    for g in (2, 5, 9):
        out = O.toy_sd(M, K, tT, tD, 200, 25, g, seed=8, flags=O.FLAG_NO_BONUS)
        assert np.array_equal(out[1], ref[1]) and np.array_equal(out[0], ref[0])


# ------------------------------------------------------------- transformer
SMALL_T = CF.ModelCfg(2, 32, 2, 64, 4, 3, CF.FP32)
SMALL_D = CF.ModelCfg(1, 16, 1, 32, 4, 3, CF.FP32)


def _small_models(shift=True):
    bt = IN.model_blob(SMALL_T, 11, 0, head_gain=6.0)
    bd = IN.model_blob(SMALL_D, 11, 1, head_gain=6.0)
    if shift:
        bd = IN.shift_blob(SMALL_D, bd, **{"head.b_mu": 0.4, "head.b_s": -0.2,
                                           "head.b_k2": np.array([0.5, 0.0, -0.5])})
    return bt, bd


def _hist(B, H, K, seed):
    rng = np.random.default_rng(seed)
    return (rng.exponential(1.0, (B, H)).astype(np.float32),
            rng.integers(0, K, (B, H)).astype(np.int32))


@pytest.mark.slow
def test_transformer_sd_equals_ar_in_distribution():
    """>= 1e5 events: SD and AR agree in law (two-sample KS on tau per
    position block, chi-square on marks), and SD passes the PIT test
    against the target's own conditional law: u = G_T(tau_i | h_{i-1}) is
    Uniform(0,1) (the time-rescaling KS of App. A.4 with the target as
    ground truth), marks match sum_i f_T(. | h_{i-1})."""
    bt, bd = _small_models()
    B, H, N, gamma = 2000, 8, 50, 4
    tau, marks = _hist(B, H, 3, 0)
    sd = O.sample_sd(SMALL_T, bt, SMALL_D, bd, tau, marks, N, gamma, seed=21)
    ar = O.sample_ar(SMALL_T, bt, tau, marks, N, seed=22)
    st = sd["stats"]
    alpha = st[:, 2].sum() / st[:, 1].sum()
    assert 0.05 < alpha < 0.95, alpha
    # one value per sequence at fixed indices: independent samples
    for j in (0, 9, 24, 49):
        assert stats.ks_2samp(sd["tau"][:, j], ar["tau"][:, j]).pvalue > P_MIN
        ct = np.stack([np.bincount(sd["k"][:, j], minlength=3), np.bincount(ar["k"][:, j], minlength=3)])
        assert stats.chi2_contingency(ct)[1] > P_MIN
    # PIT against the target's teacher-forced heads
    full_tau = np.concatenate([tau, sd["tau"].astype(np.float32)], 1)
    full_k = np.concatenate([marks, sd["k"]], 1)
    hd, _, _ = O.score(SMALL_T, bt, full_tau, full_k)
    M = SMALL_T.n_mix
    rows = hd[:, H - 1:H + N - 1].reshape(-1, hd.shape[-1])
    u = HP.pit_times(rows, M, full_tau[:, H:].ravel())
    assert stats.kstest(u, "uniform").pvalue > P_MIN
    # heads really do vary with history (otherwise index errors go unseen)
    assert rows[:, M:2 * M].std() > 0.3
    v = HP.pit_marks(rows, M, full_k[:, H:].ravel(), np.random.default_rng(0))
    assert stats.kstest(v, "uniform").pvalue > P_MIN


def test_transformer_identical_draft_equals_ar():
    bt, _ = _small_models()
    tau, marks = _hist(6, 5, 3, 1)
    ar = O.sample_ar(SMALL_T, bt, tau, marks, 40, seed=3)
    sd = O.sample_sd(SMALL_T, bt, SMALL_T, bt, tau, marks, 40, 5, seed=3)
    assert np.array_equal(ar["k"], sd["k"])
    assert np.array_equal(ar["tau"], sd["tau"]) and np.array_equal(ar["t"], sd["t"])
    assert sd["stats"][:, 1].sum() == sd["stats"][:, 2].sum()


def test_transformer_no_bonus_gamma_invariance_and_resume():
    bt, bd = _small_models()
    tau, marks = _hist(8, 6, 3, 2)
    ref = O.sample_sd(SMALL_T, bt, SMALL_D, bd, tau, marks, 30, 1, seed=4, flags=O.FLAG_NO_BONUS)
    for g in (3, 7):
        out = O.sample_sd(SMALL_T, bt, SMALL_D, bd, tau, marks, 30, g, seed=4, flags=O.FLAG_NO_BONUS)
        assert np.array_equal(out["k"], ref["k"]) and np.array_equal(out["tau"], ref["tau"])
    # resume from an emitted prefix: positions key the slots, so the
    # continuation is the same (exact up to fp32 storage of the prefix)
    n1 = 12
    tau2 = np.concatenate([tau, ref["tau"][:, :n1].astype(np.float32)], 1)
    mk2 = np.concatenate([marks, ref["k"][:, :n1]], 1)
    part = O.sample_sd(SMALL_T, bt, SMALL_D, bd, tau2, mk2, 30 - n1, 3, seed=4, flags=O.FLAG_NO_BONUS)
    agree = part["k"] == ref["k"][:, n1:]
    assert agree.mean() > 0.95
    ar = O.sample_ar(SMALL_T, bt, tau, marks, 30, seed=9)
    ar2 = O.sample_ar(SMALL_T, bt, np.concatenate([tau, ar["tau"][:, :n1].astype(np.float32)], 1),
                      np.concatenate([marks, ar["k"][:, :n1]], 1), 30 - n1, seed=9)
    assert (ar2["k"] == ar["k"][:, n1:]).mean() > 0.95


def test_single_mark_never_rejects_on_marks():
    """K = 1: f_T = f_D = 1, so a draft that differs only in its mark head
    is never rejected and SD equals AR; with K = 3 the same change causes
    mark rejections."""
    T1 = CF.ModelCfg(2, 32, 2, 64, 4, 1, CF.FP32)
    bt = IN.model_blob(T1, 5, 0, head_gain=6.0)
    bd = IN.shift_blob(T1, bt, **{"head.b_k2": 3.0, "head.b_k1": 0.7})
    tau, marks = _hist(5, 6, 1, 3)
    sd = O.sample_sd(T1, bt, T1, bd, tau, marks, 30, 4, seed=2)
    ar = O.sample_ar(T1, bt, tau, marks, 30, seed=2)
    assert sd["stats"][:, 2].sum() == sd["stats"][:, 1].sum()
    assert np.array_equal(sd["tau"], ar["tau"])
    T3 = SMALL_T
    bt3 = IN.model_blob(T3, 5, 0, head_gain=6.0)
    bd3 = IN.shift_blob(T3, bt3, **{"head.b_k2": np.array([2.0, 0.0, -2.0])})
    tau3, marks3 = _hist(5, 6, 3, 3)
    sd3 = O.sample_sd(T3, bt3, T3, bd3, tau3, marks3, 30, 4, seed=2)
    assert sd3["stats"][:, 2].sum() < sd3["stats"][:, 1].sum()
    assert sd3["stats"][:, 3].sum() == 0     # times identical: no Theorem 1 loop
