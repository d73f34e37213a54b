"""The tcgen05 form of the target's attention (TPPSD_ATTN_TC=1: keys on the
M side of both tensor-core products, TMA-staged K / V tiles, fp16 V cache
and weights, split-key flash-decoding for long contexts) against the oracle:
teacher-forced scores of every bf16 workload shape, sampling at the
workload shapes including gamma = 16 (32-row query blocks) and target-only
AR, the headline launch, the split-key path at the long-context shape, and
the reference changes of its softmax (forced by a zero slack)."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from tests import gpu_common as G

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _tc(monkeypatch):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    monkeypatch.setenv("TPPSD_ATTN_TC", "1")


def _score(tcfg, bt, B, n, K, seed=0):
    tau, mk = G.hist(B, n, K, seed)
    dcfg = CF.ModelCfg(1, 32, 2, 128, tcfg.n_mix, K, CF.BF16)
    bd = IN.model_blob(dcfg, 0, 1)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, n + 4, 2)
    hd, lg, lf = s.score(0, tau, mk)
    hd, lg, lf = hd.cpu().numpy(), lg.cpu().numpy(), lf.cpu().numpy()
    s.close()
    ohd, olg, olf = O.score(tcfg, bt, tau, mk)
    return np.abs(hd[:, :-1] - ohd[:, :-1]).max(), np.abs(lf[:, 1:] - olf[:, 1:]).max()


@pytest.mark.parametrize("idx,B,n", [(1, 3, 300), (2, 2, 300), (3, 1, 530), (4, 2, 140)])
def test_tc_attention_scores_match_oracle(idx, B, n):
    """d_head 32 (d 128 / 4 heads, d 256 / 8 heads) and 64 (d 512 / 8 heads),
    32-row query blocks over several 128-key tiles with a ragged last one."""
    wl = CF.BY_INDEX[idx]
    bt = IN.model_blob(wl.target, 0, 0)
    dh, df = _score(wl.target, bt, B, n, wl.target.n_marks)
    assert dh < G.TOL_BF16 and df < G.TOL_BF16, (dh, df)


def test_tc_attention_reference_changes(monkeypatch):
    """A zero slack makes every tile whose scores exceed the reference start
    a new accumulation segment (the path that keeps fp16 weights in range
    for real score spreads); the scores stay those of the oracle."""
    monkeypatch.setenv("TPPSD_ATTN_SLACK", "0")
    tcfg = CF.ModelCfg(2, 128, 4, 512, 8, 5, CF.BF16)
    bt = IN.model_blob(tcfg, 2, 0, head_gain=2.0)
    dh, df = _score(tcfg, bt, 2, 520, 5, seed=3)
    assert dh < G.TOL_BF16 and df < G.TOL_BF16, (dh, df)


CASES = {
    "c2_g8": (CF.C2, None, 12, 140, 32, 8),
    "c3_g16": (CF.C3, None, 8, 140, 40, 16),
    "c4_g10": (CF.C4, None, 3, 300, 32, 10),
    "c5_d64": (CF.C5, 1, 12, 140, 32, 8),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_tc_attention_sampling_matches_oracle(name):
    wl, didx, B, H, N, g = CASES[name]
    dcfg = wl.draft if didx is None else wl.drafts[didx]
    bt = IN.model_blob(wl.target, wl.seed, 0)
    bd = IN.shift_blob(dcfg, IN.model_blob(dcfg, wl.seed, 1), **{"head.b_mu": 0.3})
    tau, mk = IN.histories(wl.with_(hist_len=H), batch=B, seed=3)
    s = G.make_sampler(wl.target, dcfg, bt, bd, B, H + N + g + 4, g)
    s.prefill(tau, mk)
    gpu = G.to_np(s.sample(N, g, 41))
    st, stats = s.stats()
    ar = G.to_np(s.sample_ar(16, 43))
    s.close()
    ora = O.sample_sd(wl.target, bt, dcfg, bd, tau, mk, N, g, 41)
    ident, exc, fails = G.compare_sequences(gpu, ora, G.MARGIN_BF16, rtol=G.RTOL_BF16)
    print(f"[parity] tc attention {name}: {ident} identical, {exc} excused of {B}")
    assert not fails, fails
    assert ident >= G.min_identical(B) and st == 0
    oar = O.sample_ar(wl.target, bt, tau, mk, 16, 43)
    ident, exc, fails = G.compare_sequences(ar, oar, G.MARGIN_BF16, rtol=G.RTOL_BF16)
    assert not fails and ident >= G.min_identical(B), (ident, exc, fails)


def test_tc_attention_split_keys_long_context():
    """Two sequences with 900-event histories at the headline model shape:
    the verify and AR passes split each sequence's keys across eight CTAs
    (flash-decoding), and the last CTA of each item merges the partial
    results (the long-context shape's sampling case above splits too)."""
    wl = CF.C2
    bt = IN.model_blob(wl.target, wl.seed, 0)
    bd = IN.shift_blob(wl.draft, IN.model_blob(wl.draft, wl.seed, 1), **{"head.b_mu": 0.3})
    B, H, N, g = 2, 900, 40, 8
    tau, mk = G.hist(B, H, wl.target.n_marks, 6)
    s = G.make_sampler(wl.target, wl.draft, bt, bd, B, H + N + g + 4, g)
    s.prefill(tau, mk)
    gpu = G.to_np(s.sample(N, g, 47))
    st, _ = s.stats()
    ar = G.to_np(s.sample_ar(16, 49))
    s.close()
    ora = O.sample_sd(wl.target, bt, wl.draft, bd, tau, mk, N, g, 47)
    ident, exc, fails = G.compare_sequences(gpu, ora, G.MARGIN_BF16, rtol=G.RTOL_BF16)
    print(f"[parity] tc attention split keys: {ident} identical, {exc} excused of {B}")
    assert not fails, fails
    assert ident >= G.min_identical(B) and st == 0
    oar = O.sample_ar(wl.target, bt, tau, mk, 16, 49)
    _, _, fails = G.compare_sequences(ar, oar, G.MARGIN_BF16, rtol=G.RTOL_BF16)
    assert not fails, fails
