"""End-time stop rule (Alg. 1) and the survival term of Eq. 2 on the CUDA
path, through the C ABI, against the oracle (needs a GB300)."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from paper_2507_09252_gb300 import tppsd as T
from tests import gpu_common as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    T.load()


def _check_fill(out):
    """Slots after count[b] hold NaN times and mark -1; the kept ones are
    finite, increasing and at most t_end."""
    for b in range(out["k"].shape[0]):
        c = int(out["count"][b])
        assert np.all(np.isnan(out["t"][b, c:])) and np.all(np.isnan(out["tau"][b, c:]))
        assert np.all(out["k"][b, c:] == -1)
        assert np.all(np.isfinite(out["t"][b, :c])) and np.all(out["k"][b, :c] >= 0)


def _near_boundary(t_row, c, t_end, rtol=1e-5):
    """A count may differ only if an event sits within rtol of t_end."""
    near = np.abs(t_row - t_end) <= rtol * abs(t_end)
    return bool(np.any(near[max(c - 1, 0):c + 1]))


def _common_prefix(g, o):
    """Both runs cut to the shorter of their two kept prefixes (so a count
    difference is judged separately from the events themselves)."""
    g2 = {k: np.array(g[k], copy=True) for k in ("tau", "k")}
    o2 = {k: np.array(o[k], copy=True) for k in ("tau", "k", "margin")}
    for b in range(g2["k"].shape[0]):
        c = min(int(g["count"][b]), int(o["count"][b]))
        for d in (g2, o2):
            d["tau"][b, c:] = 1.0
            d["k"][b, c:] = 0
        o2["margin"][b, c:] = np.inf
    return g2, o2


@pytest.mark.parametrize("ar,gamma", [(False, 4), (False, 1), (True, 0)])
def test_until_matches_oracle_and_fixed_count_prefix(ar, gamma):
    """GPU vs oracle under the stop rule (sequences identical except after a
    near-tie decision, counts equal), and the GPU's kept events are bit for
    bit the prefix of its own fixed-count run."""
    tcfg, dcfg, bt, bd = G.small_models(gain=1.5)
    B, H, N = 24, 7, 80
    tau, mk = G.hist(B, H, 3, 5)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, H + N + 12, 8)
    s.prefill(tau, mk)
    if ar:
        full = G.to_np(s.sample_ar(N, 77))
    else:
        full = G.to_np(s.sample(N, gamma, 77))
    t_end = float(np.median(full["t"][:, 30]))
    if ar:
        g = G.to_np(s.sample_ar_until(t_end, N, 77))
        o = O.sample_ar_until(tcfg, bt, tau, mk, N, t_end, 77)
    else:
        g = G.to_np(s.sample_until(t_end, N, gamma, 77))
        o = O.sample_sd_until(tcfg, bt, dcfg, bd, tau, mk, N, t_end, gamma, 77)
    st, stats = s.stats()
    assert st == T.TPPSD_OK
    _check_fill(g)
    counts_full = (full["t"] <= t_end).sum(1)
    assert np.array_equal(g["count"], counts_full)
    for b in range(B):
        c = int(g["count"][b])
        assert np.array_equal(g["t"][b, :c], full["t"][b, :c])
        assert np.array_equal(g["k"][b, :c], full["k"][b, :c])
    # fewer events drawn than the fixed-count run
    assert stats["emitted"] < B * N
    g2, o2 = _common_prefix(g, o)
    ident, exc, fails = G.compare_sequences(g2, o2, G.MARGIN_FP32)
    assert not fails, fails
    assert ident >= B - 4
    for b in range(B):
        if g["count"][b] != o["count"][b]:
            i = G.first_divergence({k: g2[k][b] for k in ("tau", "k")}, {k: o2[k][b] for k in ("tau", "k")})
            assert i >= 0 or _near_boundary(o["t"][b], int(o["count"][b]), t_end), b
    assert sum(int(g["count"][b] == o["count"][b]) for b in range(B)) >= B - 4
    s.close()


def test_until_edge_cases():
    tcfg, dcfg, bt, bd = G.small_models(gain=1.5)
    B, H, N = 5, 4, 30
    tau, mk = G.hist(B, H, 3, 9)
    t_hist = tau.astype(np.float64).sum(1)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, H + N + 8, 6)
    s.prefill(tau, mk)
    # end time before every history's last event: nothing generated
    z = G.to_np(s.sample_until(float(t_hist.min()) - 1e-3, N, 3, 1))
    assert np.all(z["count"] == 0) and np.all(np.isnan(z["t"])) and np.all(z["k"] == -1)
    za = G.to_np(s.sample_ar_until(float(t_hist.min()) - 1e-3, N, 1))
    assert np.all(za["count"] == 0)
    # one history past the end time, the others not
    mid = float(np.sort(t_hist)[2])
    part = G.to_np(s.sample_until(mid, N, 3, 1))
    assert np.all(part["count"][t_hist > mid] == 0)
    # +inf is the fixed-count call
    inf = G.to_np(s.sample_until(np.inf, N, 3, 1))
    ref = G.to_np(s.sample(N, 3, 1))
    assert np.all(inf["count"] == N)
    assert all(np.array_equal(inf[k], ref[k]) for k in ("tau", "t", "k"))
    # the event cap binds before a far end time
    cap = G.to_np(s.sample_ar_until(1e12, 7, 2))
    assert np.all(cap["count"] == 7)
    # host-loop driven rounds give the same result as the graph
    t_end = float(np.median(ref["t"][:, 10]))
    a = G.to_np(s.sample_until(t_end, N, 3, 1))
    b = G.to_np(s.sample_until(t_end, N, 3, 1, flags=T.TPPSD_FLAG_HOST_LOOP))
    assert all(np.array_equal(a[k], b[k], equal_nan=k in ("tau", "t")) for k in a)
    # host (numpy) outputs, the count included
    ht = np.zeros((B, N), np.float32); htt = np.zeros((B, N)); hk = np.zeros((B, N), np.int32)
    hc = np.zeros(B, np.int32)
    T.tppsd_sample_until(s.ctx, B, t_end, N, 3, 1, 0, ht, htt, hk, hc)
    assert T.tppsd_wait(s.ctx, 10000) == T.TPPSD_OK
    assert np.array_equal(hc, a["count"]) and np.array_equal(hk, a["k"])
    assert np.array_equal(htt, a["t"], equal_nan=True)
    # NaN end time is rejected
    with pytest.raises(T.TppsdError):
        s.sample_until(float("nan"), N, 3, 1)
    s.close()


def test_until_full_size_headline_workload():
    """The benchmarked launch shape (256 sequences, up to 512 events, gamma
    8, bf16) under the stop rule: the kept events are the prefix of the
    fixed-count run with t <= T, and sampled sequences agree with the oracle."""
    wl = CF.C2
    bt, bd, tau, mk = IN.workload_inputs(wl)
    B, H, N, g = wl.batch, wl.hist_len, wl.n_events, wl.gamma
    s = G.make_sampler(wl.target, wl.draft, bt, bd, B, H + N + g + 4, g)
    s.prefill(tau, mk)
    full = G.to_np(s.sample(N, g, 2024))
    t_end = float(np.median(full["t"][:, N // 2]))
    u = G.to_np(s.sample_until(t_end, N, g, 2024))
    st, _ = s.stats()
    assert st == T.TPPSD_OK
    _check_fill(u)
    assert np.array_equal(u["count"], (full["t"] <= t_end).sum(1))
    assert u["count"].max() > 0 and u["count"].max() <= N
    for b in range(B):
        c = int(u["count"][b])
        assert np.array_equal(u["t"][b, :c], full["t"][b, :c]) and np.array_equal(u["k"][b, :c], full["k"][b, :c])
    pick = [0, 97, 255]
    o = O.sample_sd_until(wl.target, bt, wl.draft, bd, tau[pick], mk[pick], 40, t_end, g, 2024, seq_ids=pick)
    sub = {k: u[k][pick, :40] for k in ("tau", "k")}
    sub["count"] = np.minimum(u["count"][pick], 40)
    g2, o2 = _common_prefix(sub, o)
    _, _, fails = G.compare_sequences(g2, o2, G.MARGIN_BF16, rtol=2e-2)
    assert not fails, fails
    s.close()


# ------------------------------------------------------------------ survival term
@pytest.mark.parametrize("which", [0, 1])
def test_score_until_survival_matches_oracle(which):
    tcfg, dcfg, bt, bd = G.small_models(gain=1.5)
    cfg, blob = (tcfg, bt) if which == 0 else (dcfg, bd)
    B, n = 6, 40
    tau, mk = G.hist(B, n, 3, 13)
    t_last = tau.astype(np.float64).sum(1)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, n + 4, 4)
    for dt in (0.05, 1.3, 6.0):
        t_end = float(t_last.max()) + dt
        hd, lg, lf, ls = (x.cpu().numpy() for x in s.score_until(which, tau, mk, t_end))
        ref = O.score_survival(cfg, blob, tau, mk, t_end)
        assert np.all(np.abs(ls - ref) <= 2e-4 * (1 + np.abs(ref))), (ls, ref)
        assert np.all(ls <= 0)
    # per-event terms equal tppsd_score's; the extra head row is the one
    # after the last event
    _, lg0, lf0 = (x.cpu().numpy() if x is not None else None for x in s.score(which, tau, mk, heads=False))
    assert np.array_equal(lg[:, 1:], lg0[:, 1:]) and np.array_equal(lf[:, 1:], lf0[:, 1:])
    ext_tau = np.concatenate([tau, np.ones((B, 1), np.float32)], 1)
    ext_mk = np.concatenate([mk, np.zeros((B, 1), np.int32)], 1)
    oh = O.score(cfg, blob, ext_tau, ext_mk)[0]
    assert np.abs(hd[:, n - 1] - oh[:, n - 1]).max() < G.TOL_FP32 * 10
    # a window ending before the last event has no survival term
    _, _, _, ls0 = s.score_until(which, tau, mk, float(t_last.min()) - 1.0)
    assert np.all(ls0.cpu().numpy() == 0.0)
    # a single event: only the survival term
    _, lg1, _, ls1 = s.score_until(which, tau[:, :1], mk[:, :1], float(tau[:, 0].max()) + 0.5)
    ref1 = O.score_survival(cfg, blob, tau[:, :1], mk[:, :1], float(tau[:, 0].max()) + 0.5)
    assert np.all(np.abs(ls1.cpu().numpy() - ref1) <= 2e-4 * (1 + np.abs(ref1)))
    assert np.all(np.isnan(lg1.cpu().numpy()))
    s.close()


def test_score_until_bf16_and_tail():
    """bf16 target of the headline shape: survival term within the bf16
    tolerance of the oracle, including windows far into the tail."""
    wl = CF.C2
    bt = IN.model_blob(wl.target, wl.seed, 0)
    bd = IN.model_blob(wl.draft, wl.seed, 1)
    tau, mk = IN.histories(wl, 4)
    s = G.make_sampler(wl.target, wl.draft, bt, bd, 4, tau.shape[1] + 4, 2)
    t_last = tau.astype(np.float64).sum(1)
    for dt in (0.5, 20.0, 400.0):
        t_end = float(t_last.max()) + dt
        _, _, _, ls = s.score_until(0, tau, mk, t_end, heads=False)
        ls = ls.cpu().numpy()
        ref = O.score_survival(wl.target, bt, tau, mk, t_end)
        assert np.all(np.isfinite(ls))
        assert np.all(np.abs(ls - ref) <= G.TOL_BF16 * (1 + np.abs(ref))), (dt, ls, ref)
    s.close()
