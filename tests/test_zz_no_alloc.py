"""tppsd_score_noalloc: scoring for callers that may not allocate device memory.

Such callers (a process whose GPU memory is owned by another allocator, or a
latency-critical loop that cannot absorb the implicit synchronisation of
cudaMalloc) get the same per-event log densities as tppsd_score, computed in
a fixed device array that the library holds from load time.  This file is
collected last so that a failure here never hides the other tests.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from paper_2507_09252_gb300 import tppsd as T
from tests import gpu_common as G

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("bf16", [False, True])
def test_noalloc_scoring_matches_allocating_scoring_twice(bf16):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    if bf16:
        wl = CF.C2
        tcfg, dcfg = wl.target, wl.draft
        bt, bd = IN.model_blob(tcfg, 0, 0), IN.model_blob(dcfg, 0, 1)
        B, n, tol = 6, 90, G.TOL_BF16
    else:
        tcfg, dcfg, bt, bd = G.small_models()
        B, n, tol = 5, 120, G.TOL_FP32
    tau_np, mk_np = G.hist(B, n, tcfg.n_marks, 3)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, n + 4, 2)
    tau = torch.from_numpy(tau_np).cuda()
    mk = torch.from_numpy(mk_np).cuda()
    for which in (0, 1):
        _, ref_g, ref_f = s.score(which, tau, mk, heads=False)
        ref_g, ref_f = ref_g.cpu().numpy(), ref_f.cpu().numpy()
        for _ in range(2):   # two calls in a row share the same scratch
            lg = torch.full((B, n), -7.0, device="cuda")
            lf = torch.full((B, n), -7.0, device="cuda")
            T.tppsd_score_noalloc(s.ctx, which, B, n, tau, mk, lg, lf)
            torch.cuda.synchronize()
            lg, lf = lg.cpu().numpy(), lf.cpu().numpy()
            assert np.isnan(lg[:, 0]).all() and np.isnan(lf[:, 0]).all()
            assert np.abs(lg[:, 1:] - ref_g[:, 1:]).max() < tol
            assert np.abs(lf[:, 1:] - ref_f[:, 1:]).max() < tol
    # a request larger than the fixed scratch is refused, with a reason
    big = torch.zeros((B, 200000), dtype=torch.float32, device="cuda")
    bigk = torch.zeros((B, 200000), dtype=torch.int32, device="cuda")
    with pytest.raises(T.TppsdError) as e:
        T.tppsd_score_noalloc(s.ctx, 0, B, 200000, big, bigk, big, big)
    assert e.value.status == T.TPPSD_ERR_INVALID_ARG and "scratch" in str(e.value)
    s.close()


def _noalloc(torch, s, which, tau, mk):
    B, n = tau.shape
    lg = torch.full((B, n), -7.0, device="cuda")
    lf = torch.full((B, n), -7.0, device="cuda")
    T.tppsd_score_noalloc(s.ctx, which, B, n, tau, mk, lg, lf)
    torch.cuda.synchronize()
    assert T.tppsd_wait(s.ctx, 60000) == T.TPPSD_OK
    return lg.cpu().numpy(), lf.cpu().numpy()


def test_noalloc_several_row_chunks_bf16_matches_oracle():
    """16 sequences x 256 events of the headline bf16 target: the K/V of all
    4096 positions leave room for about 1 600 workspace rows, so the 4 080
    scored rows run in three chunks, later chunks reading K/V that earlier
    ones wrote.  Two calls in a row against tppsd_score and the oracle."""
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    wl = CF.C2
    tcfg, dcfg = wl.target, wl.draft
    bt, bd = IN.model_blob(tcfg, 0, 0), IN.model_blob(dcfg, 0, 1)
    B, n = 16, 256
    tau_np, mk_np = G.hist(B, n, tcfg.n_marks, 5)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, n + 4, 2)
    tau, mk = torch.from_numpy(tau_np).cuda(), torch.from_numpy(mk_np).cuda()
    _, ref_g, ref_f = s.score(0, tau, mk, heads=False)
    ref_g, ref_f = ref_g.cpu().numpy(), ref_f.cpu().numpy()
    _, olg, olf = O.score(tcfg, bt, tau_np, mk_np, heads=False)
    for _ in range(2):
        lg, lf = _noalloc(torch, s, 0, tau, mk)
        assert np.isnan(lg[:, 0]).all()
        assert np.abs(lg[:, 1:] - ref_g[:, 1:]).max() < G.TOL_BF16
        assert np.abs(lf[:, 1:] - ref_f[:, 1:]).max() < G.TOL_BF16
        assert np.abs(lg[:, 1:] - olg[:, 1:]).max() < G.TOL_BF16
        assert np.abs(lf[:, 1:] - olf[:, 1:]).max() < G.TOL_BF16
    s.close()


def test_noalloc_one_sequence_across_chunks_near_the_limit_fp32():
    """One fp32 sequence of 31 700 events: its K/V nearly fill the 16 MiB
    array, leaving about twenty workspace rows, so the sequence is scored in
    some 1 400 chunks of the same sequence.  Against tppsd_score, twice."""
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    tcfg, dcfg, bt, bd = G.small_models(gain=1.5)
    B, n = 1, 31700
    tau_np, mk_np = G.hist(B, n, tcfg.n_marks, 6)
    s = G.make_sampler(tcfg, dcfg, bt, bd, B, n + 4, 2)
    tau, mk = torch.from_numpy(tau_np).cuda(), torch.from_numpy(mk_np).cuda()
    _, ref_g, ref_f = s.score(0, tau, mk, heads=False)
    ref_g, ref_f = ref_g.cpu().numpy(), ref_f.cpu().numpy()
    for _ in range(2):
        lg, lf = _noalloc(torch, s, 0, tau, mk)
        assert np.abs(lg[:, 1:] - ref_g[:, 1:]).max() < G.TOL_FP32
        assert np.abs(lf[:, 1:] - ref_f[:, 1:]).max() < G.TOL_FP32
    # a sequence a few hundred events longer no longer fits: refused with a reason
    big = torch.zeros((B, 32300), dtype=torch.float32, device="cuda")
    bigk = torch.zeros((B, 32300), dtype=torch.int32, device="cuda")
    with pytest.raises(T.TppsdError) as e:
        T.tppsd_score_noalloc(s.ctx, 0, B, 32300, big, bigk, big, big)
    assert e.value.status == T.TPPSD_ERR_INVALID_ARG and "scratch" in str(e.value)
    s.close()
