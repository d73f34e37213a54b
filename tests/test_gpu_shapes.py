"""Sampling parity at the shapes of every bf16 workload (Alg. 1 over the full
verify path, against the oracle), beyond the headline one: d = 256 and 512
targets with 6 and 8 layers, 8 heads of 32 and 64 dimensions, 2-layer d64
and d128 drafts (whose draft KV stays in HBM), the c5 d32 draft, gamma up to
16 (17 verify rows per sequence), and target-only AR at the long-context
shape.  Drafts have a shifted b_mu so that rejections, Theorem-1 resampling
and mark residual draws all happen; histories are drawn from each
workload's own recipe and are longer than one 128-key attention tile."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from tests import gpu_common as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


CASES = {
    # name: (workload, draft index or None, batch, history, events, gamma)
    "c3_g8": (CF.C3, None, 12, 140, 32, 8),
    "c3_g16": (CF.C3, None, 8, 140, 40, 16),
    "c4_g10": (CF.C4, None, 3, 300, 32, 10),
    "c5_d32": (CF.C5, 0, 12, 140, 32, 8),
    "c5_d64": (CF.C5, 1, 12, 140, 32, 8),
    "c5_d128": (CF.C5, 2, 8, 140, 32, 8),
}


def _models(wl, didx):
    dcfg = wl.draft if didx is None else wl.drafts[didx]
    bt = IN.model_blob(wl.target, wl.seed, 0)
    bd = IN.shift_blob(dcfg, IN.model_blob(dcfg, wl.seed, 1), **{"head.b_mu": 0.3})
    return wl.target, dcfg, bt, bd


@pytest.mark.parametrize("name", sorted(CASES))
def test_sequence_parity_bf16_workload_shapes(name):
    wl, didx, B, H, N, g = CASES[name]
    tcfg, dcfg, bt, bd = _models(wl, didx)
    tau, mk = IN.histories(wl.with_(hist_len=H), batch=B, seed=3)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, H + N + g + 4, g)
    s.prefill(tau, mk)
    gpu = G.to_np(s.sample(N, g, 41))
    st, stats = s.stats()
    s.close()
    ora = O.sample_sd(tcfg, bt, dcfg, bd, tau, mk, N, g, 41)
    ident, exc, fails = G.compare_sequences(gpu, ora, G.MARGIN_BF16, rtol=G.RTOL_BF16)
    print(f"[parity] {name}: {ident} identical, {exc} excused of {B}; "
          f"accepted {stats['accepted']}/{stats['drafted']}, resample iters {stats['resample_iters']}")
    assert not fails, fails
    assert ident >= G.min_identical(B), (ident, exc, B)
    assert st == 0 and stats["accepted"] < stats["drafted"] and stats["resample_iters"] > 0


def test_autoregressive_parity_long_context_shape():
    """Target-only AR (one query row per sequence) at the d = 512, 8-layer
    shape over a 300-event history."""
    wl = CF.C4
    tcfg, dcfg, bt, bd = _models(wl, None)
    B, H, N = 8, 300, 24
    tau, mk = IN.histories(wl.with_(hist_len=H), batch=B, seed=4)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, H + N + 4, 1)
    s.prefill(tau, mk)
    gpu = G.to_np(s.sample_ar(N, 43))
    s.close()
    ora = O.sample_ar(tcfg, bt, tau, mk, N, 43)
    ident, exc, fails = G.compare_sequences(gpu, ora, G.MARGIN_BF16, rtol=G.RTOL_BF16)
    print(f"[parity] c4 AR: {ident} identical, {exc} excused of {B}")
    assert not fails, fails
    assert ident >= G.min_identical(B)
