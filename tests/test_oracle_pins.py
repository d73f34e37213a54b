"""Pins of the CPU oracle against what the paper and the mathematics fix.

No test here compares the oracle with itself: each checks it against a
published vector, a closed form, a library routine, an invariant, or a law
derived in App. A.
"""
import os

import numpy as np
import pytest
from scipy import integrate, stats

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from tests import helpers as HP

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- Philox
def test_philox_known_answers():
    """Philox4x32-10 against the Random123 known-answer vectors (SC'11)."""
    rows = [l.split() for l in open(os.path.join(GOLDEN, "philox4x32_10_kat.txt"))
            if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        out = O.philox4x32(v[0:4], v[4:6])
        assert list(out) == v[6:10]


def test_uniforms_open_interval_and_moments():
    u = np.array([O.uniforms(123, s, p, b) for s in range(4) for p in range(500) for b in range(5)])
    u = u.ravel()
    assert u.min() > 0.0 and u.max() < 1.0
    # exact 24-bit grid values (k + 0.5) / 2^24
    k = u * 2 ** 24 - 0.5
    assert np.all(k == np.round(k))
    assert stats.kstest(u, "uniform").pvalue > 1e-3
    assert abs(np.corrcoef(u[:-1], u[1:])[0, 1]) < 0.02


def test_uniform_slots_are_distinct_streams():
    a = O.uniforms(5, 0, 10, 0)
    assert not np.array_equal(a, O.uniforms(5, 1, 10, 0))   # sequence
    assert not np.array_equal(a, O.uniforms(5, 0, 11, 0))   # position
    assert not np.array_equal(a, O.uniforms(5, 0, 10, 1))   # block
    assert not np.array_equal(a, O.uniforms(6, 0, 10, 0))   # seed
    assert not np.array_equal(O.uniforms(1, 0, 0, 0), O.uniforms(1 << 32, 0, 0, 0))  # seed hi word


# ---------------------------------------------------------------- bf16
def test_round_bf16_matches_torch():
    import torch
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.normal(0, 1, 2000), rng.normal(0, 1e-3, 500), rng.normal(0, 50, 500)])
    x = x.astype(np.float32).astype(np.float64)   # fp32 inputs: torch's rounding is exact RNE
    ref = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
    got = np.array([O.round_bf16(v) for v in x])
    assert np.array_equal(got, ref)
    # ties go to even: 1 + 2^-8 is halfway between 1 and 1 + 2^-7
    assert O.round_bf16(1.0 + 2.0 ** -8) == 1.0
    assert O.round_bf16(1.0 + 3 * 2.0 ** -8) == 1.0 + 2.0 ** -6


# ---------------------------------------------------------------- encoding
@pytest.mark.parametrize("d", [16, 32, 128])
def test_temporal_encoding_properties(d):
    """App. D.4 (THP): z(0) = (0,1,0,1,...), each (sin, cos) pair on the unit
    circle, the first pair is (sin t, cos t), frequencies fall geometrically
    by 10000^(-2/D) per pair."""
    z0 = O.temporal_encoding(d, 0.0)
    assert np.allclose(z0[0::2], 0.0) and np.allclose(z0[1::2], 1.0)
    t = 3.7
    z = O.temporal_encoding(d, t)
    assert np.allclose(z[0::2] ** 2 + z[1::2] ** 2, 1.0, atol=1e-14)
    assert abs(z[0] - np.sin(t)) < 1e-15 and abs(z[1] - np.cos(t)) < 1e-15
    # recover each pair's frequency from small-t phases
    ts = 1e-3
    zs = O.temporal_encoding(d, ts)
    omega = np.arctan2(zs[0::2], zs[1::2]) / ts
    ratio = omega[1:] / omega[:-1]
    assert np.allclose(ratio, 10000.0 ** (-2.0 / d), rtol=1e-6)
    # absolute time: large t still exact (no fp32 loss)
    zb = O.temporal_encoding(d, 7000.25)
    assert abs(zb[0] - np.sin(7000.25)) < 1e-12


# ---------------------------------------------------------------- heads
@pytest.mark.parametrize("M", [1, 4, 16])
def test_log_g_matches_scipy_and_integrates_to_one(M):
    """log g equals the log of scipy's log-normal mixture pdf and integrates
    to 1 by quadrature in log tau (Sec. 4.2 density, App. A.1)."""
    rng = np.random.default_rng(M)
    for rep in range(3):
        hd = HP.random_head(rng, M, 3)
        taus = np.exp(rng.normal(0, 2, 50))
        ref = np.log(HP.mixture_pdf(hd, M, taus))
        got = O.log_g(M, hd, taus)
        assert np.allclose(got, ref, atol=1e-10, rtol=1e-10)
        f = lambda x: np.exp(O.log_g(M, hd, np.exp(x))[0] + x)
        val, err = integrate.quad(f, -40, 40, limit=400, epsabs=1e-12)
        assert abs(val - 1.0) < 1e-6


@pytest.mark.parametrize("M,K", [(1, 1), (4, 5), (8, 22)])
def test_direct_sampler_matches_closed_form(M, K):
    """z ~ Cat(w), eps ~ N(0,1), tau = exp(mu_z + sigma_z eps) (App. A.1):
    the draws follow G(tau) = sum_m w_m Phi((log tau - mu_m)/sigma_m) (KS),
    and marks follow f (chi-square)."""
    rng = np.random.default_rng(10 + M)
    hd = HP.random_head(rng, M, K)
    n = 100000
    tau, k = O.sample_head(M, K, hd, n, seed=99)
    assert stats.kstest(tau, lambda x: HP.mixture_cdf(hd, M, x)).pvalue > 1e-3
    f = np.exp(hd[3 * M:])
    assert HP.chi2_pvalue(np.bincount(k, minlength=K), n * f) > 1e-3 if K > 1 else np.all(k == 0)
    # closed-form mean sum_m w_m exp(mu_m + sigma_m^2 / 2)
    w = np.exp(hd[:M]); mu = hd[M:2 * M]; sg = np.exp(hd[2 * M:3 * M])
    if sg.max() < 0.8:
        mean = (w * np.exp(mu + sg ** 2 / 2)).sum()
        assert abs(tau.mean() / mean - 1) < 0.02


def test_theorem1_resampler_matches_residual_density():
    """Theorem 1: propose from g_T, accept with max(0, g_T - g_D)/g_T gives
    g' = norm(max(0, g_T - g_D)) (Eq. 3).  KS against g' integrated by
    quadrature; mean iterations 1/Z (Z = total-variation mass)."""
    rng = np.random.default_rng(3)
    M = 4
    hT = HP.random_head(rng, M, 2)
    hD = hT.copy()
    hD[M:2 * M] += 0.6
    hD[2 * M:3 * M] -= 0.2
    cdf, Z = HP.residual_cdf_factory(hT, hD, M)
    n = 40000
    tau, it = O.resample_time(M, hT, hD, n, seed=7)
    assert stats.kstest(tau, cdf).pvalue > 1e-3
    assert abs(it.mean() * Z - 1) < 0.03
    # must NOT look like g_T itself (that would be the biased rule App. A.2 warns about)
    assert stats.kstest(tau, lambda x: HP.mixture_cdf(hT, M, x)).pvalue < 1e-6


def test_mark_residual_matches_eq4():
    rng = np.random.default_rng(4)
    M, K = 2, 6
    hT = HP.random_head(rng, M, K)
    hD = HP.random_head(rng, M, K)
    n = 60000
    k = O.resample_mark(M, K, hT, hD, n, seed=11)
    r = np.maximum(0, np.exp(hT[3 * M:]) - np.exp(hD[3 * M:]))
    assert HP.chi2_pvalue(np.bincount(k, minlength=K), n * r / r.sum()) > 1e-3
    assert np.all(r[k] > 0)


# ---------------------------------------------------------------- model
@pytest.mark.parametrize("wl", [CF.C1, CF.C2])
def test_model_heads_match_torch_library_transformer(wl):
    """Encoder (Sec. 4.2; post-LN reading) and heads against
    torch.nn.TransformerEncoderLayer + F.linear in float64, fp32 models.
    bf16 rounding is off here (dtype forced to fp32) so only the model
    definition is compared."""
    tgt = CF.ModelCfg(**{**wl.target.__dict__, "dtype": CF.FP32})
    blob = IN.model_blob(tgt, 0, 0)
    rng = np.random.default_rng(1)
    B, n = 3, 40
    tau = rng.exponential(1.0, (B, n)).astype(np.float32)
    marks = rng.integers(0, tgt.n_marks, (B, n)).astype(np.int32)
    hd, lg, lf = O.score(tgt, blob, tau, marks)
    ref = HP.torch_reference_heads(tgt, blob, tau, marks)
    assert np.allclose(hd[:, :-1], ref[:, :-1], atol=1e-9, rtol=1e-9)
    # per-event log densities agree with the heads they come from
    M = tgt.n_mix
    i = 17
    assert abs(lg[1, i + 1] - np.log(HP.mixture_pdf(ref[1, i], M, float(tau[1, i + 1])))) < 1e-9
    assert abs(lf[1, i + 1] - ref[1, i, 3 * M + marks[1, i + 1]]) < 1e-9


def test_attention_with_zero_qk_is_causal_mean():
    """With the Q and K weights zeroed (biases are zero too) every score is
    equal, so the attention output at position i is the plain mean of the
    values v_j over positions j = 0..i.  The layer is rebuilt here in numpy
    with that closed form in place of attention (THP encoding of App. D.4,
    post-LN layer, heads of Sec. 4.2 by library F.linear); a wrong causal
    bound, normaliser or head split in the oracle's attention fails it."""
    cfg = CF.ModelCfg(1, 16, 2, 32, 3, 4, CF.FP32)
    blob = IN.model_blob(cfg, 5, 0)
    offs = IN.blob_offsets(cfg)
    d = cfg.d_model

    def P(name):
        o, shape = offs[name]
        return blob[o:o + int(np.prod(shape))].reshape(shape).astype(np.float64)

    o, _ = offs["layer0.w_qkv"]
    blob[o:o + 2 * d * d] = 0.0                       # W_q and W_k rows
    assert not P("layer0.b_qkv")[:2 * d].any()         # zero biases: every score is 0
    rng = np.random.default_rng(2)
    B, n = 2, 12
    tau = rng.exponential(1.0, (B, n)).astype(np.float32)
    marks = rng.integers(0, cfg.n_marks, (B, n)).astype(np.int32)
    hd, _, _ = O.score(cfg, blob, tau, marks)

    t = np.cumsum(tau.astype(np.float64), 1)
    j = np.arange(d)
    ang = t[..., None] / 10000.0 ** ((j - j % 2) / d)
    x = np.where(j % 2 == 1, np.cos(ang), np.sin(ang)) + P("type_emb")[marks]
    wqkv, bqkv = P("layer0.w_qkv"), P("layer0.b_qkv")
    v = x @ wqkv[2 * d:].T + bqkv[2 * d:]
    a = np.cumsum(v, 1) / np.arange(1, n + 1)[None, :, None]   # causal mean of V

    def ln(y, g, b):
        mu = y.mean(-1, keepdims=True)
        var = ((y - mu) ** 2).mean(-1, keepdims=True)
        return (y - mu) / np.sqrt(var + 1e-5) * g + b

    h1 = ln(x + a @ P("layer0.w_o").T + P("layer0.b_o"), P("layer0.ln1_g"), P("layer0.ln1_b"))
    f = np.maximum(h1 @ P("layer0.w_1").T + P("layer0.b_1"), 0.0) @ P("layer0.w_2").T + P("layer0.b_2")
    h2 = ln(h1 + f, P("layer0.ln2_g"), P("layer0.ln2_b"))
    ref = HP.torch_heads(cfg, blob, h2)
    assert np.allclose(hd[:, :-1], ref[:, :-1], atol=1e-10)


def test_cached_equals_recompute():
    """KV-cached encoding and full re-encoding after every rollback agree
    (the rollback of Alg. 1 is a length reset)."""
    wl = CF.C1.with_(batch=2, n_events=24)
    bt, bd, tau, marks = IN.workload_inputs(wl)
    bd = IN.shift_blob(wl.draft, bd, **{"head.b_mu": 0.5})
    a = O.sample_sd(wl.target, bt, wl.draft, bd, tau, marks, wl.n_events, wl.gamma, 3)
    b = O.sample_sd(wl.target, bt, wl.draft, bd, tau, marks, wl.n_events, wl.gamma, 3, recompute=True)
    assert np.array_equal(a["k"], b["k"])
    assert np.allclose(a["tau"], b["tau"], rtol=1e-12)
    assert a["stats"][:, 2].sum() < a["stats"][:, 1].sum()   # some rejections happened
