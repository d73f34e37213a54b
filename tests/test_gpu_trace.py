"""TPPSD_FLAG_DEBUG_TRACE: the recorded verify decisions are consistent with
the sampled sequences and with the oracle's decision margins (needs a GB300)."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import tppsd as T
from tests import gpu_common as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    T.load()


def _blocks(codes, rounds):
    """Split one sequence's trace into rounds: (round id, codes) in order."""
    out = []
    for c, r in zip(codes, rounds):
        if out and out[-1][0] == r:
            out[-1][1].append(c)
        else:
            out.append((r, [c]))
    return out


@pytest.mark.parametrize("gamma,flags,dtype", [(4, 0, CF.FP32), (7, 0, CF.FP32),
                                               (4, T.TPPSD_FLAG_NO_BONUS, CF.FP32), (4, 0, CF.BF16)])
def test_trace_decisions(gamma, flags, dtype):
    tcfg, dcfg, bt, bd = G.small_models(gain=1.5, dtype=dtype)
    B, N = 24, 60
    tau, mk = G.hist(B, 7, 3, 5)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, 7 + N + gamma + 2, 8)
    s.prefill(tau, mk)
    g = G.to_np(s.sample(N, gamma, 77, flags | T.TPPSD_FLAG_DEBUG_TRACE))
    tr = s.trace(B, N)
    # a later untraced call must not leave a stale trace readable
    s.prefill(tau, mk)
    s.sample(4, gamma, 78, flags)
    with pytest.raises(T.TppsdError):
        s.trace(1, 1)
    s.close()
    o = O.sample_sd(tcfg, bt, dcfg, bd, tau, mk, N, gamma, 77, flags=flags)

    mt, mkk, code, rnd = tr[..., 0], tr[..., 1], tr[..., 2].astype(int), tr[..., 3].astype(int)
    assert set(np.unique(code)) <= {1, 2, 4, 6, 8}, np.unique(code)
    acc = code == 1
    assert np.all(mt[acc] < 0) and np.all(mkk[acc] < 0)
    tested = (code & 6) != 0
    assert np.all((mt[tested] >= 0) == ((code[tested] & 2) != 0))
    assert np.all((mkk[tested] >= 0) == ((code[tested] & 4) != 0))
    bonus = code == 8
    assert np.all(np.isnan(mt[bonus])) and np.all(np.isnan(mkk[bonus]))
    if flags & T.TPPSD_FLAG_NO_BONUS:
        assert not bonus.any()
    # every round: a run of accepted drafts closed by one rejection or the
    # bonus (a round with all gamma drafts accepted and no bonus is open);
    # only the last round may be cut by the event budget
    rounds_gpu = 0
    for b in range(B):
        blocks = _blocks(code[b], rnd[b])
        rounds_gpu += len(blocks)
        ids = [r for r, _ in blocks]
        assert ids == sorted(set(ids)), ids
        for i, (_, cs) in enumerate(blocks):
            assert all(c == 1 for c in cs[:-1])
            last = i == len(blocks) - 1
            assert len(cs) <= gamma + 1
            if cs[-1] == 1:
                assert last or (flags & T.TPPSD_FLAG_NO_BONUS and len(cs) == gamma)
            if not last:
                assert len(cs) == (gamma if cs[-1] == 1 else len(cs))
    margin = G.MARGIN_FP32 if dtype == CF.FP32 else G.MARGIN_BF16
    rtol = 1e-4 if dtype == CF.FP32 else G.RTOL_BF16
    # a test margin's own error: r = exp(log-density difference) in fp32
    # (about 1e-5 of r) or from bf16 weights (about 1e-2 of r)
    m_err = 1e-3 if dtype == CF.FP32 else 5e-2
    # divergences from the oracle come only after a near-tie decision, by the
    # oracle's margins or by the GPU's own
    _, _, fails = G.compare_sequences(g, o, margin, rtol=rtol, gpu_trace=tr)
    assert not fails, fails
    ident = 0
    for b in range(B):
        if G.first_divergence({k: g[k][b] for k in ("tau", "k")}, {k: o[k][b] for k in ("tau", "k")}, rtol) >= 0:
            continue
        ident += 1
        # same sequence, same rounds: the oracle counts every round it ran
        assert len(_blocks(code[b], rnd[b])) == o["stats"][b, 0], b
        n_acc = int(acc[b].sum())
        assert n_acc <= o["stats"][b, 2] <= n_acc + gamma
        # the oracle's smallest decision margin at an event bounds the GPU's
        # test margins there, up to the GPU's own rounding
        m = np.minimum(np.abs(mt[b]), np.abs(mkk[b]))
        ok = np.isnan(m) | (o["margin"][b] <= m + m_err)
        assert ok.all(), (b, np.nonzero(~ok)[0][:5])
    assert ident >= G.min_identical(B) // 2
