"""Failure paths of the C ABI on the GPU, all made on the host side or by a
wait that nothing completes (no kernel is made to fault or hang):

  * the Theorem-1 loop stopped by a lowered iteration cap
    (TPPSD_WARN_RESAMPLE_CAP, reading c6 of the sampler);
  * the device round loop of Alg. 1 stopped by a lowered round cap
    (TPPSD_ERR_ROUND_LIMIT);
  * the host watchdog tppsd_wait giving up on a long call (TPPSD_ERR_TIMEOUT);
  * a bounded mbarrier wait inside a tensor-core kernel running out: the
    kernel records the timeout and returns, the call reports
    TPPSD_ERR_TIMEOUT, and the context keeps working.
"""
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


def _mismatched(B=24, H=7, N=60, gamma=4):
    tcfg, dcfg, bt, bd = G.small_models(gain=1.5)
    tau, mk = G.hist(B, H, 3, 5)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, H + N + gamma + 4, gamma)
    s.prefill(tau, mk)
    return s, (tcfg, dcfg, bt, bd, tau, mk)


@pytest.mark.parametrize("flags", [0, T.TPPSD_FLAG_HOST_LOOP])
def test_resample_cap_reported_and_restored(flags):
    s, (tcfg, dcfg, bt, bd, tau, mk) = _mismatched()
    T.tppsd_set_limits(s.ctx, 1, 0)            # one proposal per Theorem-1 loop
    out = G.to_np(s.sample(60, 4, 77, flags))
    st, stats = T.tppsd_get_stats(s.ctx)
    assert st == T.TPPSD_WARN_RESAMPLE_CAP and stats["cap_hits"] > 0
    assert stats["resample_iters"] >= stats["cap_hits"]
    assert np.isfinite(out["tau"]).all() and (out["tau"] > 0).all()
    T.tppsd_set_limits(s.ctx, 0, 0)            # back to the default cap
    g = G.to_np(s.sample(60, 4, 77, flags))
    st, stats = T.tppsd_get_stats(s.ctx)
    assert st == T.TPPSD_OK and stats["cap_hits"] == 0
    o = O.sample_sd(tcfg, bt, dcfg, bd, tau, mk, 60, 4, 77)
    _, _, fails = G.compare_sequences(g, o, G.MARGIN_FP32)
    assert not fails, fails
    s.close()


@pytest.mark.parametrize("flags", [0, T.TPPSD_FLAG_HOST_LOOP])
def test_round_limit_reported_and_restored(flags):
    s, _ = _mismatched()
    T.tppsd_set_limits(s.ctx, 0, 3)            # far fewer rounds than 60 events need
    s.sample(60, 4, 5, flags)
    with pytest.raises(T.TppsdError) as e:
        T.tppsd_get_stats(s.ctx)
    assert e.value.status == T.TPPSD_ERR_ROUND_LIMIT
    T.tppsd_set_limits(s.ctx, 0, 0)
    s.sample(60, 4, 5, flags)
    st, stats = T.tppsd_get_stats(s.ctx)
    assert st == T.TPPSD_OK and stats["emitted"] >= 24 * 60
    with pytest.raises(T.TppsdError):
        T.tppsd_set_limits(s.ctx, -1, 0)
    s.close()


def test_host_watchdog_times_out_on_a_long_call():
    """tppsd_wait with a zero limit right after enqueueing the headline call
    (about 15 ms of GPU work) returns TPPSD_ERR_TIMEOUT; a later wait with
    room returns OK and the output is complete."""
    import torch
    wl = CF.C2
    bt, bd, tau, mk = IN.workload_inputs(wl)
    B, H, N, g = wl.batch, wl.hist_len, wl.n_events, wl.gamma
    s = G.make_sampler(wl.target, wl.draft, bt, bd, B, H + N + g + 4, g)
    s.prefill(tau, mk)
    out = s._outputs(B, N)
    torch.cuda.synchronize()
    T.tppsd_sample(s.ctx, B, N, g, 3, 0, *out)
    assert T.tppsd_wait(s.ctx, 0) == T.TPPSD_ERR_TIMEOUT
    assert "timed out" in T.tppsd_last_error(s.ctx)
    assert T.tppsd_wait(s.ctx, 60000) == T.TPPSD_OK
    assert torch.isfinite(out[0]).all() and (out[2] >= 0).all()
    s.close()


def test_bounded_pipeline_wait_runs_out_and_context_recovers(monkeypatch):
    """TPPSD_FAULT=wait: the tensor-core QKV GEMM waits on a barrier that
    nothing completes; its bounded wait runs out, the kernel records the
    timeout and returns, and the scoring call reports TPPSD_ERR_TIMEOUT.
    Without the variable the same context scores correctly again."""
    tcfg = CF.ModelCfg(2, 128, 4, 512, 8, 5, CF.BF16)
    dcfg = CF.ModelCfg(1, 32, 2, 128, 8, 5, CF.BF16)
    bt, bd = IN.model_blob(tcfg, 4, 0), IN.model_blob(dcfg, 4, 1)
    tau, mk = G.hist(2, 40, 5, 7)
    s = G.make_sampler(tcfg, dcfg, bt, bd, 2, 48, 2)
    monkeypatch.setenv("TPPSD_FAULT", "wait")
    s.score(0, tau, mk, heads=False)
    assert T.tppsd_wait(s.ctx, 60000) == T.TPPSD_ERR_TIMEOUT
    assert "wait timed out" in T.tppsd_last_error(s.ctx)
    monkeypatch.delenv("TPPSD_FAULT")
    _, lg, lf = s.score(0, tau, mk, heads=False)
    assert T.tppsd_wait(s.ctx, 60000) == T.TPPSD_OK
    _, olg, olf = O.score(tcfg, bt, tau, mk, heads=False)
    assert np.abs(lg.cpu().numpy()[:, 1:] - olg[:, 1:]).max() < G.TOL_BF16
    assert np.abs(lf.cpu().numpy()[:, 1:] - olf[:, 1:]).max() < G.TOL_BF16
    s.close()
