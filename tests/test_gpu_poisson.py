"""TPP-SD with the Poisson draft of App. D.3 on the CUDA path, through the C
ABI, against the oracle (needs a GB300)."""
import numpy as np
import pytest
from scipy import stats

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from paper_2507_09252_gb300 import tppsd as T
from paper_2507_09252_gb300.sampler import fit_poisson_draft
from tests import gpu_common as G
from tests import helpers as HP

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    T.load()


LAM, P3 = 1.1, np.array([0.45, 0.35, 0.2])


@pytest.mark.parametrize("gamma,flags", [(4, 0), (1, 0), (7, 0), (4, T.TPPSD_FLAG_NO_BONUS)])
def test_poisson_draft_parity_fp32(gamma, flags):
    """Sequences identical to the oracle except after a near-tie decision;
    with no excused sequence the acceptance and Theorem-1 counts agree."""
    tcfg, dcfg, bt, bd = G.small_models(gain=1.5)
    B, H, N = 24, 7, 60
    tau, mk = G.hist(B, H, 3, 5)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, H + N + 12, 8)
    s.prefill(tau, mk)
    g = G.to_np(s.sample_poisson(N, gamma, LAM, P3, 77, flags))
    st, stats_ = s.stats()
    s.close()
    o = O.sample_sd_poisson(tcfg, bt, tau, mk, N, gamma, LAM, P3, 77, flags=flags)
    assert st == T.TPPSD_OK
    ident, exc, fails = G.compare_sequences(g, o, G.MARGIN_FP32)
    assert not fails, fails
    assert ident >= B - 4
    assert stats_["accepted"] < stats_["drafted"] and stats_["resample_iters"] > 0
    assert stats_["draft_keys"] == 0
    if exc == 0:
        assert stats_["accepted"] == o["stats"][:, 2].sum()
        assert stats_["rounds"] == o["stats"][:, 0].sum()
        assert stats_["resample_iters"] == o["stats"][:, 3].sum()


def test_poisson_draft_until_and_edge_cases():
    tcfg, dcfg, bt, bd = G.small_models(gain=1.5)
    B, H, N = 16, 6, 70
    tau, mk = G.hist(B, H, 3, 8)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, H + N + 12, 8)
    s.prefill(tau, mk)
    full = G.to_np(s.sample_poisson(N, 5, LAM, P3, 3))
    t_end = float(np.median(full["t"][:, 25]))
    u = G.to_np(s.sample_poisson_until(t_end, N, 5, LAM, P3, 3))
    assert np.array_equal(u["count"], (full["t"] <= t_end).sum(1))
    for b in range(B):
        c = int(u["count"][b])
        assert np.array_equal(u["t"][b, :c], full["t"][b, :c]) and np.array_equal(u["k"][b, :c], full["k"][b, :c])
        assert np.all(np.isnan(u["t"][b, c:])) and np.all(u["k"][b, c:] == -1)
    o = O.sample_sd_poisson_until(tcfg, bt, tau, mk, N, t_end, 5, LAM, P3, 3)
    assert (u["count"] == o["count"]).sum() >= B - 3
    # unnormalised probabilities are normalised; host loop = graph
    a = G.to_np(s.sample_poisson(N, 5, LAM, 4 * P3, 3))
    assert all(np.array_equal(a[k], full[k]) for k in a)
    h = G.to_np(s.sample_poisson(N, 5, LAM, P3, 3, flags=T.TPPSD_FLAG_HOST_LOOP))
    assert all(np.array_equal(h[k], full[k]) for k in h)
    # a zero-probability mark is never drafted; the target may still emit it
    z = G.to_np(s.sample_poisson(N, 5, LAM, np.array([0.5, 0.5, 0.0]), 3))
    assert np.isfinite(z["tau"]).all()
    for bad_rate, bad_p in ((0.0, P3), (-2.0, P3), (np.nan, P3), (LAM, np.array([0.5, -0.1, 0.6])),
                            (LAM, np.zeros(3))):
        with pytest.raises(T.TppsdError):
            s.sample_poisson(N, 5, bad_rate, bad_p, 3)
    s.close()


def test_poisson_draft_distribution_bf16_headline_shape():
    """Headline target (bf16, 256 sequences x 512 events, gamma 8) with the
    MLE Poisson draft fitted on a pilot AR sample of the target (the data a
    trained target models): PIT of the output against the GPU target's
    teacher-forced heads is Uniform(0,1), rejections happen, and sampled
    rows agree with the oracle on their prefix."""
    wl = CF.C2
    tcfg, dcfg = wl.target, wl.draft
    bt, bd = IN.model_blob(tcfg, wl.seed, 0), IN.model_blob(dcfg, wl.seed, 1)
    tau, mk = IN.histories(wl)
    B, H, N, g = wl.batch, wl.hist_len, wl.n_events, wl.gamma
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, H + N + g + 4, g)
    s.prefill(tau, mk)
    pilot = G.to_np(s.sample_ar(64, 7))
    rate, probs = fit_poisson_draft(pilot["tau"], pilot["k"], tcfg.n_marks)
    sd = G.to_np(s.sample_poisson(N, g, rate, probs, 41))
    st, stats_ = s.stats()
    assert st == T.TPPSD_OK
    assert np.isfinite(sd["tau"]).all() and (sd["tau"] > 0).all()
    assert 0.05 < stats_["accepted"] / stats_["drafted"] < 0.98 and stats_["resample_iters"] > 0
    pick = [0, 130, 255]
    o = O.sample_sd_poisson(tcfg, bt, tau[pick], mk[pick], 40, g, rate, probs, 41, seq_ids=pick)
    sub = {k: sd[k][pick, :40] for k in ("tau", "k")}
    _, _, fails = G.compare_sequences(sub, o, G.MARGIN_BF16, rtol=2e-2)
    assert not fails, fails
    full_tau = np.concatenate([tau, sd["tau"]], 1)
    full_k = np.concatenate([mk, sd["k"]], 1)
    hd, _, _ = s.score(0, full_tau, full_k)
    hd = hd.cpu().numpy()
    s.close()
    M = tcfg.n_mix
    rows = hd[:, H - 1:H + N - 1].reshape(-1, hd.shape[-1]).astype(np.float64)
    rng = np.random.default_rng(2)
    assert stats.kstest(HP.pit_times(rows, M, full_tau[:, H:].ravel()), "uniform").pvalue > 1e-3
    assert stats.kstest(HP.pit_marks(rows, M, full_k[:, H:].ravel(), rng), "uniform").pvalue > 1e-3
