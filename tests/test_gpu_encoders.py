"""SAHP and AttNHP encoders (App. D.4) on the CUDA path, through the C ABI,
against the oracle (needs a GB300)."""
import numpy as np
import pytest
from scipy import stats

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from paper_2507_09252_gb300 import tppsd as T
from tests import gpu_common as G
from tests import helpers as HP
from tests.test_gpu_parity import _score_case

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    T.load()


def _models(enc, dtype=CF.FP32, gain=1.5, tcfg=None, dcfg=None, seed=11):
    tcfg = tcfg or CF.ModelCfg(2, 32, 2, 64, 4, 3, dtype, enc)
    dcfg = dcfg or CF.ModelCfg(1, 16, 1, 32, 4, 3, dtype, enc)
    bt = IN.model_blob(tcfg, seed, 0, head_gain=gain)
    bd = IN.model_blob(dcfg, seed, 1, head_gain=gain)
    bd = IN.shift_blob(dcfg, bd, **{"head.b_mu": 0.4, "head.b_s": -0.2,
                                    "head.b_k2": np.linspace(0.5, -0.5, dcfg.n_marks)})
    return tcfg, dcfg, bt, bd


@pytest.mark.parametrize("enc", [CF.SAHP, CF.ATTNHP])
def test_score_parity_fp32(enc):
    tcfg, dcfg, bt, bd = _models(enc, gain=6.0)
    _score_case(tcfg, dcfg, bt, bd, 5, 150, 3, G.TOL_FP32)


@pytest.mark.parametrize("enc", [CF.SAHP, CF.ATTNHP])
def test_score_parity_bf16_tensor_core_shapes(enc):
    """d = 128 targets (tensor-core QKV over [z | h] rows for AttNHP, the
    fused cluster block for SAHP) and a d = 32 draft, several row tiles."""
    tcfg = CF.ModelCfg(2, 128, 4, 512, 8, 5, CF.BF16, enc)
    dcfg = CF.ModelCfg(1, 32, 2, 128, 8, 5, CF.BF16, enc)
    bt, bd = IN.model_blob(tcfg, 3, 0, head_gain=2.0), IN.model_blob(dcfg, 3, 1)
    _score_case(tcfg, dcfg, bt, bd, 2, 300, 5, G.TOL_BF16)


@pytest.mark.parametrize("enc,gamma", [(CF.SAHP, 4), (CF.ATTNHP, 4), (CF.ATTNHP, 1)])
def test_sequence_parity_fp32(enc, gamma):
    tcfg, dcfg, bt, bd = _models(enc)
    tau, mk = G.hist(24, 7, 3, 5)
    N = 60
    s = G.make_sampler(tcfg, dcfg, bt, bd, 24, 7 + N + 12, 8)
    s.prefill(tau, mk)
    g = G.to_np(s.sample(N, gamma, 77))
    st, stats_ = s.stats()
    ar = G.to_np(s.sample_ar(N, 78))
    s.close()
    o = O.sample_sd(tcfg, bt, dcfg, bd, tau, mk, N, gamma, 77)
    oa = O.sample_ar(tcfg, bt, tau, mk, N, 78)
    assert st == T.TPPSD_OK
    ident, exc, fails = G.compare_sequences(g, o, G.MARGIN_FP32)
    assert not fails, fails
    assert ident >= 20
    _, _, fails_ar = G.compare_sequences(ar, oa, G.MARGIN_FP32)
    assert not fails_ar, fails_ar
    assert stats_["accepted"] < stats_["drafted"] and stats_["resample_iters"] > 0
    if exc == 0:
        assert stats_["accepted"] == o["stats"][:, 2].sum()


def test_attnhp_headline_shape_distribution():
    """c2-shaped AttNHP models (bf16 target 4 x d128, draft 1 x d32), 256 x 512
    events: PIT of the SD output against the GPU target's teacher-forced
    heads, and oracle agreement on the prefix of three rows."""
    wl = CF.C2
    tcfg = CF.ModelCfg(**{**wl.target.__dict__, "encoder": CF.ATTNHP})
    dcfg = CF.ModelCfg(**{**wl.draft.__dict__, "encoder": CF.ATTNHP})
    bt, bd = IN.model_blob(tcfg, wl.seed, 0), IN.model_blob(dcfg, wl.seed, 1)
    tau, mk = IN.histories(wl)
    B, H, N, g = wl.batch, wl.hist_len, wl.n_events, wl.gamma
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, H + N + g + 4, g)
    s.prefill(tau, mk)
    sd = G.to_np(s.sample(N, g, 51))
    st, stats_ = s.stats()
    assert st == T.TPPSD_OK and np.isfinite(sd["tau"]).all()
    assert stats_["accepted"] < stats_["drafted"]
    pick = [0, 128, 255]
    o = O.sample_sd(tcfg, bt, dcfg, bd, tau[pick], mk[pick], 40, g, 51, seq_ids=pick)
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
    rng = np.random.default_rng(3)
    assert stats.kstest(HP.pit_times(rows, M, full_tau[:, H:].ravel()), "uniform").pvalue > 1e-3
    assert stats.kstest(HP.pit_marks(rows, M, full_k[:, H:].ravel(), rng), "uniform").pvalue > 1e-3


def test_attnhp_draft_outside_the_team_kernel_is_refused():
    tcfg = CF.ModelCfg(2, 32, 2, 64, 4, 3, CF.FP32, CF.ATTNHP)
    dcfg = CF.ModelCfg(1, 64, 1, 64, 4, 3, CF.FP32, CF.ATTNHP)   # d/heads = 64
    bt, bd = IN.model_blob(tcfg, 0, 0), IN.model_blob(dcfg, 0, 1)
    with pytest.raises(T.TppsdError):
        G.make_sampler(tcfg, dcfg, bt, bd, 2, 40, 4)
