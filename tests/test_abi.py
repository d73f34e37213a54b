"""The C-ABI library builds, loads and exports every declared symbol; host-side
argument checks and injected faults work without a GPU."""
import os
import re
import subprocess
import sys

import numpy as np
import pytest

from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from paper_2507_09252_gb300 import tppsd as T

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "tppsd.h")).read()
    return sorted(set(re.findall(r"\b(tppsd_[a-z_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol():
    L = T.load()
    names = _declared()
    assert "tppsd_sample" in names and "tppsd_prefill" in names and len(names) >= 11
    for n in names:
        assert hasattr(L, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", T.lib_path()], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (tppsd_\w+)", out))
    assert set(names) <= exported


@pytest.mark.parametrize("wl", CF.BY_INDEX)
def test_blob_size_agrees_with_generator(wl):
    for cfg in (wl.target, wl.draft) + tuple(wl.drafts):
        assert T.tppsd_blob_floats(cfg) == IN.blob_size(cfg) == IN.model_blob(cfg, 0, 0).size
        for enc in (CF.SAHP, CF.ATTNHP):
            c = CF.ModelCfg(**{**cfg.__dict__, "encoder": enc})
            assert T.tppsd_blob_floats(c) == IN.blob_size(c)
    small = CF.ModelCfg(2, 32, 2, 64, 4, 3, CF.BF16)
    for enc in (CF.SAHP, CF.ATTNHP):
        c = CF.ModelCfg(**{**small.__dict__, "encoder": enc})
        assert T.tppsd_blob_floats(c) == IN.model_blob(c, 0, 0).size
    bad = CF.ModelCfg(**{**wl.target.__dict__, "encoder": 3})
    assert T.tppsd_blob_floats(bad) == 0


def test_invalid_shapes_rejected():
    bad = CF.ModelCfg(2, 30, 2, 64, 4, 1, 0)      # d not a multiple of 16
    assert T.tppsd_blob_floats(bad) == 0
    bad = CF.ModelCfg(2, 32, 3, 64, 4, 1, 0)      # heads do not divide d
    assert T.tppsd_blob_floats(bad) == 0
    bad = CF.ModelCfg(2, 32, 2, 64, 65, 1, 0)     # too many components
    assert T.tppsd_blob_floats(bad) == 0


def _try_create(**kw):
    wl = CF.C1
    bt = IN.model_blob(wl.target, 0, 0)
    bd = IN.model_blob(wl.draft, 0, 1)
    args = dict(target=wl.target, draft=wl.draft, target_blob=bt, draft_blob=bd,
                max_batch=4, max_positions=100, max_gamma=4)
    args.update(kw)
    return T.tppsd_create_models(**args)


def test_argument_errors_before_any_device_work():
    with pytest.raises(T.TppsdError) as e:
        _try_create(max_batch=0)
    assert e.value.status == T.TPPSD_ERR_INVALID_ARG
    with pytest.raises(T.TppsdError) as e:
        _try_create(max_gamma=40)
    assert e.value.status == T.TPPSD_ERR_INVALID_ARG
    wl = CF.C1
    with pytest.raises(T.TppsdError) as e:   # mark spaces differ
        _try_create(draft=CF.ModelCfg(1, 16, 1, 32, 4, 3, 0),
                    draft_blob=IN.model_blob(CF.ModelCfg(1, 16, 1, 32, 4, 3, 0), 0, 1))
    assert e.value.status == T.TPPSD_ERR_INVALID_ARG
    # null context
    assert T.load().tppsd_prefill(None, 1, None, None, 1, None) == T.TPPSD_ERR_INVALID_ARG
    assert T.load().tppsd_sample(None, 1, 1, 1, 0, 0, None, None, None, None) == T.TPPSD_ERR_INVALID_ARG
    assert T.status_str(T.TPPSD_ERR_ROUND_LIMIT) == "round limit reached"


def test_injected_allocation_failure():
    code = ("import sys; sys.path.insert(0, %r)\n"
            "from tests.test_abi import _try_create\n"
            "from paper_2507_09252_gb300 import tppsd as T\n"
            "try:\n    _try_create()\nexcept T.TppsdError as e:\n    print('STATUS', e.status)\n") % ROOT
    env = dict(os.environ, TPPSD_FAULT="alloc")
    out = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, cwd=ROOT)
    assert f"STATUS {T.TPPSD_ERR_OOM}" in out.stdout, out.stdout + out.stderr


def test_no_device_is_reported_not_crashed():
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(T.TppsdError) as e:
        _try_create()
    assert e.value.status == T.TPPSD_ERR_NO_DEVICE


def test_poisson_draft_fit_is_the_mle():
    """tppsd_fit_poisson_draft (App. D.3): rate = events / observed time,
    mark probabilities = frequencies.  Pinned by the likelihood itself: the
    Poisson log-likelihood n log(rate) - rate * sum(T_b) is stationary at the
    fitted rate and lower on both sides of it; on a homogeneous Poisson
    sample the fit recovers the true rate.  Host arrays, so no GPU is needed."""
    from paper_2507_09252_gb300.sampler import fit_poisson_draft
    rng = np.random.default_rng(0)
    tau = rng.exponential(1 / 2.5, (200, 50)).astype(np.float32)
    mk = rng.choice(3, size=(200, 50), p=[0.6, 0.3, 0.1]).astype(np.int32)
    rate, p = fit_poisson_draft(tau, mk, 4)
    T_obs = tau.astype(np.float64).sum()
    assert rate == pytest.approx(tau.size / T_obs, rel=1e-12)
    assert abs(rate - 2.5) < 0.1
    assert np.allclose(p[:3], np.bincount(mk.ravel(), minlength=3) / mk.size) and p[3] == 0.0

    def loglik(lam, T_tot):
        return tau.size * np.log(lam) - lam * T_tot

    for T_tot in (T_obs, T_obs + 300.0):
        win = None if T_tot == T_obs else tau.astype(np.float64).sum(1) + 1.5
        r, _ = fit_poisson_draft(tau, mk, 4, t_window=win)
        assert loglik(r, T_tot) > loglik(r * 1.01, T_tot) and loglik(r, T_tot) > loglik(r * 0.99, T_tot)
        assert abs(tau.size / r - T_tot) < 1e-6 * T_tot          # d/dlam loglik = 0
    # invalid inputs
    with pytest.raises(T.TppsdError):
        fit_poisson_draft(tau, mk, 2)                              # mark 2 out of range
    with pytest.raises(T.TppsdError):
        fit_poisson_draft(tau, mk, 4, t_window=np.zeros(200))      # window before the last event
    with pytest.raises(T.TppsdError):
        fit_poisson_draft(-tau, mk, 4)                             # negative times
