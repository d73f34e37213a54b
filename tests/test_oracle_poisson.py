"""Oracle pins for TPP-SD with the Poisson draft of App. D.3: a homogeneous
Poisson process (rate lambda) drafts the times and marks are drafted iid
from p.  Checked against the exponential law itself, Theorem 1's residual
density by quadrature, the exact Markov law of a toy target, gamma
invariance without the bonus event, and AR sampling in law."""
import numpy as np
import pytest
from scipy import stats

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from tests import helpers as HP

P_MIN = 1e-3
SMALL_T = CF.ModelCfg(2, 32, 2, 64, 4, 3, CF.FP32)


def test_poisson_draws_are_exponential_and_p():
    lam, p = 2.5, np.array([0.2, 0.0, 0.5, 0.3])
    n = 60000
    tau, k = O.sample_poisson(lam, p, n, seed=4)
    assert stats.kstest(tau, stats.expon(scale=1 / lam).cdf).pvalue > P_MIN
    assert abs(tau.mean() * lam - 1) < 0.02
    assert HP.chi2_pvalue(np.bincount(k, minlength=4), n * p) > P_MIN
    assert np.all(k != 1)                           # zero probability: never drawn
    tau3, k3 = O.sample_poisson(lam, 3 * p, n, seed=4)   # p is normalised
    assert np.array_equal(k3, k) and np.array_equal(tau3, tau)
    for bad_lam, bad_p in ((0.0, p), (-1.0, p), (lam, [0.5, -0.1]), (lam, [0.0, 0.0])):
        with pytest.raises(ValueError):
            O.sample_poisson(bad_lam, bad_p, 10, seed=1)


def test_theorem1_against_poisson_draft_matches_residual_density():
    """Theorem 1 with g_D(tau) = lam exp(-lam tau): accepted proposals follow
    norm(max(0, g_T - g_D)); KS against its quadrature CDF (scipy's
    log-normal and exponential densities), mean iterations 1/Z."""
    rng = np.random.default_rng(8)
    M, lam = 3, 0.8
    hT = HP.random_head(rng, M, 1)[:3 * M]
    x = np.linspace(-14.0, 10.0, 240001)
    tt = np.exp(x)
    r = np.maximum(0.0, HP.mixture_pdf(hT, M, tt) - stats.expon(scale=1 / lam).pdf(tt)) * tt
    c = np.concatenate([[0.0], np.cumsum(0.5 * (r[1:] + r[:-1]) * np.diff(x))])
    Z = c[-1]
    n = 40000
    tau, it = O.resample_time_poisson(M, hT, lam, n, seed=5)
    assert stats.kstest(tau, lambda t: np.interp(np.log(t), x, c / Z)).pvalue > P_MIN
    assert abs(it.mean() * Z - 1) < 0.03
    assert stats.kstest(tau, lambda t: HP.mixture_cdf(hT, M, t)).pvalue < 1e-6


def _toy_tables(rng, M, K):
    return np.stack([HP.random_head(rng, M, K) for _ in range(K)])


def _markov_law(table, M, K, n):
    f = np.exp(table[:, 3 * M:])
    law = {(): 1.0}
    for _ in range(n):
        law = {seq + (k,): q * f[seq[-1] if seq else 0, k] for seq, q in law.items() for k in range(K)}
    return law


@pytest.mark.parametrize("gamma,flags", [(1, 0), (3, 0), (3, O.FLAG_NO_BONUS)])
def test_toy_sd_poisson_matches_exact_markov_law(gamma, flags):
    """Toy target with K = 3 marks, Poisson draft: the law of (k1, k2, k3)
    is the product of the target's transitions (exact enumeration), times
    pass the PIT against g_T(. | previous mark), and both kinds of
    rejection happen."""
    rng = np.random.default_rng(42)
    M, K, N, B = 3, 3, 3, 100000
    tT = _toy_tables(rng, M, K)
    lam, p = 1.3, np.array([0.5, 0.3, 0.2])
    tau, k, st = O.toy_sd_poisson(M, K, tT, lam, p, B, N, gamma, seed=19, flags=flags)
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
    acc = st[:, 2].sum() / st[:, 1].sum()
    assert 0.05 < acc < 0.95
    assert st[:, 3].sum() > 0


def _target():
    return IN.model_blob(SMALL_T, 11, 0, head_gain=6.0)


def _hist(B, H, K, seed):
    rng = np.random.default_rng(seed)
    return (rng.exponential(1.0, (B, H)).astype(np.float32),
            rng.integers(0, K, (B, H)).astype(np.int32))


def test_poisson_no_bonus_gamma_invariance_and_until_prefix():
    """Without the bonus every position is decided by its own slots, so the
    output does not depend on gamma; the end-time form keeps the t <= T
    prefix of the fixed-count run."""
    bt = _target()
    tau, mk = _hist(8, 6, 3, 2)
    lam, p = 1.1, np.array([0.4, 0.35, 0.25])
    ref = O.sample_sd_poisson(SMALL_T, bt, tau, mk, 30, 1, lam, p, seed=4, flags=O.FLAG_NO_BONUS)
    for g in (3, 8):
        out = O.sample_sd_poisson(SMALL_T, bt, tau, mk, 30, g, lam, p, seed=4, flags=O.FLAG_NO_BONUS)
        assert np.array_equal(out["k"], ref["k"]) and np.array_equal(out["tau"], ref["tau"])
    assert ref["stats"][:, 2].sum() < ref["stats"][:, 1].sum()
    full = O.sample_sd_poisson(SMALL_T, bt, tau, mk, 60, 4, lam, p, seed=6)
    t_end = float(np.median(full["t"][:, 20]))
    until = O.sample_sd_poisson_until(SMALL_T, bt, tau, mk, 60, t_end, 4, lam, p, seed=6)
    for b in range(8):
        c = int((full["t"][b] <= t_end).sum())
        assert until["count"][b] == c
        assert np.array_equal(until["t"][b, :c], full["t"][b, :c])
        assert np.array_equal(until["k"][b, :c], full["k"][b, :c])


@pytest.mark.slow
def test_transformer_sd_poisson_equals_ar_in_law():
    """>= 1e5 events from the Poisson-draft sampler: per-index two-sample
    tests against AR over independent sequences, and the PIT of times and
    marks against the target's teacher-forced heads."""
    bt = _target()
    B, H, N, gamma = 2000, 8, 50, 6
    tau, mk = _hist(B, H, 3, 0)
    lam, p = 0.9, np.array([0.5, 0.3, 0.2])
    sd = O.sample_sd_poisson(SMALL_T, bt, tau, mk, N, gamma, lam, p, seed=31)
    ar = O.sample_ar(SMALL_T, bt, tau, mk, N, seed=32)
    st = sd["stats"]
    alpha = st[:, 2].sum() / st[:, 1].sum()
    assert 0.05 < alpha < 0.95, alpha
    for j in (0, 9, 24, 49):
        assert stats.ks_2samp(sd["tau"][:, j], ar["tau"][:, j]).pvalue > P_MIN
        ct = np.stack([np.bincount(sd["k"][:, j], minlength=3), np.bincount(ar["k"][:, j], minlength=3)])
        assert stats.chi2_contingency(ct)[1] > P_MIN
    full_tau = np.concatenate([tau, sd["tau"].astype(np.float32)], 1)
    full_k = np.concatenate([mk, sd["k"]], 1)
    hd, _, _ = O.score(SMALL_T, bt, full_tau, full_k)
    M = SMALL_T.n_mix
    rows = hd[:, H - 1:H + N - 1].reshape(-1, hd.shape[-1])
    u = HP.pit_times(rows, M, full_tau[:, H:].ravel())
    assert stats.kstest(u, "uniform").pvalue > P_MIN
    v = HP.pit_marks(rows, M, full_k[:, H:].ravel(), np.random.default_rng(0))
    assert stats.kstest(v, "uniform").pvalue > P_MIN
