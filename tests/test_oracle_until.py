"""Oracle pins for the end-time stop rule (Alg. 1: sample until the end time
T, keep the events in [0, T]) and the survival term of the log-likelihood
(Sec. 3.1, Eq. 2)."""
import numpy as np
import pytest
from scipy import integrate, stats

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from tests import helpers as HP

TCFG = CF.ModelCfg(2, 32, 2, 64, 4, 3, CF.FP32)
DCFG = CF.ModelCfg(1, 16, 1, 32, 4, 3, CF.FP32)


def _models(gain=1.5):
    bt = IN.model_blob(TCFG, 5, 0, head_gain=gain)
    bd = IN.model_blob(DCFG, 5, 1, head_gain=gain)
    bd = IN.shift_blob(DCFG, bd, **{"head.b_mu": 0.3, "head.b_k2": np.linspace(0.4, -0.4, 3)})
    return bt, bd


def _hist(B, H, seed=1):
    rng = np.random.default_rng(seed)
    return (rng.exponential(1.0, (B, H)).astype(np.float32),
            rng.integers(0, 3, (B, H)).astype(np.int32))


@pytest.mark.parametrize("M", [1, 4])
def test_survival_matches_quadrature_of_the_density(M):
    """log S(u) = log of the integral of g from u to infinity (quadrature in
    log tau, independent of the closed-form CDF), also deep in the tail."""
    rng = np.random.default_rng(20 + M)
    for _ in range(3):
        hd = HP.random_head(rng, M, 2)
        for u in (0.05, 0.7, 2.0, 9.0):
            f = lambda x: np.exp(O.log_g(M, hd, np.exp(x))[0] + x)
            val, _ = integrate.quad(f, np.log(u), 60, limit=400, epsabs=1e-14, epsrel=1e-10)
            assert abs(O.log_survival(M, hd, u) - np.log(val)) < 1e-7
    # tail: finite, decreasing, consistent with the single-component closed form
    hd1 = np.array([0.0, 0.0, np.log(0.5), 0.0, 0.0])  # M = 1: mu 0, sigma 0.5, K = 2
    for u in (1e3, 1e8, 1e30):
        ref = stats.norm.logsf(np.log(u) / 0.5)
        assert abs(O.log_survival(1, hd1, u) - ref) < 1e-3 * abs(ref)
    vals = [O.log_survival(1, hd1, u) for u in (1.0, 10.0, 1e3, 1e10)]
    assert all(a > b for a, b in zip(vals, vals[1:]))
    assert O.log_survival(1, hd1, 0.0) == 0.0


@pytest.mark.parametrize("gamma", [1, 4])
def test_sd_until_is_the_prefix_of_the_fixed_count_run(gamma):
    """Stopping at T changes no random slot of the events before the
    crossing: the events kept are exactly those of the fixed-count run with
    t <= T."""
    bt, bd = _models()
    tau, mk = _hist(6, 8)
    N = 200
    full = O.sample_sd(TCFG, bt, DCFG, bd, tau, mk, N, gamma, seed=3)
    t_end = float(np.median(full["t"][:, 40]))
    until = O.sample_sd_until(TCFG, bt, DCFG, bd, tau, mk, N, t_end, gamma, seed=3)
    for b in range(6):
        keep = full["t"][b] <= t_end
        c = int(keep.sum())
        assert until["count"][b] == c
        assert np.array_equal(until["t"][b, :c], full["t"][b, :c])
        assert np.array_equal(until["k"][b, :c], full["k"][b, :c])
        assert np.all(np.isnan(until["t"][b, c:])) and np.all(until["k"][b, c:] == -1)
    ar_full = O.sample_ar(TCFG, bt, tau, mk, N, seed=3)
    ar = O.sample_ar_until(TCFG, bt, tau, mk, N, t_end, seed=3)
    for b in range(6):
        c = int((ar_full["t"][b] <= t_end).sum())
        assert ar["count"][b] == c
        assert np.array_equal(ar["t"][b, :c], ar_full["t"][b, :c])


def test_until_edge_cases():
    bt, bd = _models()
    tau, mk = _hist(3, 5)
    t_hist = np.cumsum(tau.astype(np.float64), axis=1)
    # end time before the last history event: nothing is generated
    r = O.sample_sd_until(TCFG, bt, DCFG, bd, tau, mk, 10, float(t_hist[:, -1].min()) - 1e-3, 3, seed=1)
    assert np.all(r["count"] == 0)
    # +inf: the fixed-count run
    r = O.sample_sd_until(TCFG, bt, DCFG, bd, tau, mk, 12, np.inf, 3, seed=1)
    f = O.sample_sd(TCFG, bt, DCFG, bd, tau, mk, 12, 3, seed=1)
    assert np.all(r["count"] == 12) and np.array_equal(r["t"], f["t"])
    # the event cap binds before the end time
    r = O.sample_ar_until(TCFG, bt, tau, mk, 7, 1e9, seed=2)
    assert np.all(r["count"] == 7)


def test_sd_until_count_law_equals_ar():
    """The number of events in (t_H, T] has the same law under TPP-SD as
    under AR sampling (two-sample chi-square on the count histogram)."""
    bt, bd = _models()
    B = 1500
    tau, mk = _hist(B, 4, seed=7)
    t0 = np.cumsum(tau.astype(np.float64), axis=1)[:, -1]
    # one common horizon: histories of equal total length
    tau = tau / t0[:, None].astype(np.float32) * 4.0
    t_end = 4.0 + 6.0
    sd = O.sample_sd_until(TCFG, bt, DCFG, bd, tau, mk, 400, t_end, 4, seed=11,
                           seq_ids=np.arange(B))
    ar = O.sample_ar_until(TCFG, bt, tau, mk, 400, t_end, seed=12, seq_ids=np.arange(B) + B)
    assert sd["count"].max() < 400 and ar["count"].max() < 400
    hi = int(max(sd["count"].max(), ar["count"].max())) + 1
    edges = np.unique(np.quantile(np.concatenate([sd["count"], ar["count"]]), np.linspace(0, 1, 9)))
    edges[-1] = hi
    a, _ = np.histogram(sd["count"], edges)
    b, _ = np.histogram(ar["count"], edges)
    _, p, _, _ = stats.chi2_contingency(np.stack([a, b]) + 0.5)
    assert p > 1e-3


def test_score_survival_matches_head_after_last_event():
    """oracle_score_survival = log S from the head the scorer gives after
    the last event (teacher forcing one event further)."""
    bt, _ = _models()
    tau, mk = _hist(4, 12, seed=3)
    t_end = float(np.cumsum(tau.astype(np.float64), axis=1)[:, -1].max()) + 0.8
    lS = O.score_survival(TCFG, bt, tau, mk, t_end)
    # heads after event i come from scoring a sequence one event longer
    ext_tau = np.concatenate([tau, np.ones((4, 1), np.float32)], axis=1)
    ext_mk = np.concatenate([mk, np.zeros((4, 1), np.int32)], axis=1)
    heads = O.score(TCFG, bt, ext_tau, ext_mk)[0]
    t_last = np.cumsum(tau.astype(np.float64), axis=1)[:, -1]
    for b in range(4):
        ref = O.log_survival(TCFG.n_mix, heads[b, 11], t_end - t_last[b])
        assert abs(lS[b] - ref) < 1e-12
