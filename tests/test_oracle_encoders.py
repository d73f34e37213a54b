"""Oracle pins for the SAHP and AttNHP history encoders (App. D.4).

SAHP: its temporal encoding is a set of sinusoids of frequency w_j (the
learned vector in the blob) with phases fixed at t = 0; its layers are the
THP layers, checked against torch.nn.TransformerEncoderLayer fed with the
oracle's SAHP encoding.  AttNHP: its encoding has the THP structure with the
wavelengths m (5M/m)^{j/D}; its layer (q, k, v from [1; z; h], attention
normalised by 1 + sum f, residual tanh) is pinned by closed forms: zero
value weights leave h = z + W k at every layer, zero query / key weights
give f = 1 and a = (sum of v) / (n + 1), and one event gives
a = sigmoid(q k / sqrt(d_head)) v.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as Fn

from oracle import oracle as O
from paper_2507_09252_gb300 import configs as CF
from paper_2507_09252_gb300 import inputs as IN
from tests import helpers as HP

SAHP_T = CF.ModelCfg(2, 32, 2, 64, 4, 3, CF.FP32, CF.SAHP)
ATT_T = CF.ModelCfg(2, 32, 2, 64, 4, 3, CF.FP32, CF.ATTNHP)


def _hist(B, n, K, seed):
    rng = np.random.default_rng(seed)
    return (rng.exponential(1.0, (B, n)).astype(np.float32),
            rng.integers(0, K, (B, n)).astype(np.int32))


def _offs(cfg):
    return IN.blob_offsets(cfg)


def _set(cfg, blob, name, value):
    o, shape = _offs(cfg)[name]
    b = blob.copy()
    b[o:o + int(np.prod(shape))] = np.broadcast_to(np.asarray(value, np.float32), shape).ravel()
    return b


def _get(cfg, blob, name):
    o, shape = _offs(cfg)[name]
    return blob[o:o + int(np.prod(shape))].reshape(shape).astype(np.float64)


# ------------------------------------------------------------------ SAHP
def test_sahp_encoding_is_sinusoids_of_the_learned_frequencies():
    blob = IN.model_blob(SAHP_T, 3, 0)
    w = _get(SAHP_T, blob, "tenc_w")
    t, dt = 37.25, 0.61
    z = O.model_temporal_encoding(SAHP_T, blob, t)
    zp = O.model_temporal_encoding(SAHP_T, blob, t + dt)
    zm = O.model_temporal_encoding(SAHP_T, blob, t - dt)
    # a sinusoid of angular frequency w: z(t+dt) + z(t-dt) = 2 cos(w dt) z(t)
    assert np.allclose(zp + zm, 2 * np.cos(w * dt) * z, atol=1e-12)
    assert np.all(np.abs(z) <= 1.0)
    # phases at t = 0 do not depend on w; with w = 0 the encoding is constant
    b0 = _set(SAHP_T, blob, "tenc_w", 0.0)
    z0 = O.model_temporal_encoding(SAHP_T, b0, 0.0)
    assert np.array_equal(z0, O.model_temporal_encoding(SAHP_T, blob, 0.0))
    assert np.allclose(O.model_temporal_encoding(SAHP_T, b0, 123.0), z0, atol=0)
    assert z0[0] == 0.0                      # phase of dimension 0 is 0 / 10000^0
    # the phases differ from THP's (which are all 0): odd dims are not all 1
    assert not np.allclose(z0[1::2], 1.0)


def test_sahp_model_matches_torch_library_layers():
    """SAHP = THP layers on the SAHP encoding: torch's
    TransformerEncoderLayer fed with the oracle's SAHP encoding."""
    blob = IN.model_blob(SAHP_T, 5, 0, head_gain=3.0)
    blob = _set(SAHP_T, blob, "tenc_w", np.linspace(-0.3, 0.4, SAHP_T.d_model))
    tau, mk = _hist(3, 20, 3, 1)
    t = np.cumsum(tau.astype(np.float64), axis=1)
    z = np.stack([[O.model_temporal_encoding(SAHP_T, blob, x) for x in row] for row in t])
    ref = HP.torch_reference_heads(SAHP_T, blob, tau, mk, z=z)
    hd = O.score(SAHP_T, blob, tau, mk)[0]
    assert np.abs(hd[:, :-1] - ref[:, :-1]).max() < 1e-9
    # and the encoding matters: THP's heads differ
    thp = CF.ModelCfg(**{**SAHP_T.__dict__, "encoder": CF.THP})
    hthp = HP.torch_reference_heads(thp, blob[:IN.blob_size(thp)], tau, mk)
    assert np.abs(hthp[:, :-1] - ref[:, :-1]).max() > 1e-3


# ------------------------------------------------------------------ AttNHP
@pytest.mark.parametrize("d", [16, 64])
def test_attnhp_encoding_structure(d):
    cfg = CF.ModelCfg(1, d, 1, 2 * d, 2, 2, CF.FP32, CF.ATTNHP)
    blob = IN.model_blob(cfg, 0, 0)
    m, M = _get(cfg, blob, "tenc_scales")
    z0 = O.model_temporal_encoding(cfg, blob, 0.0)
    assert np.allclose(z0[0::2], 0.0) and np.allclose(z0[1::2], 1.0)
    t = 3.7
    z = O.model_temporal_encoding(cfg, blob, t)
    assert np.allclose(z[0::2] ** 2 + z[1::2] ** 2, 1.0, atol=1e-14)
    # first pair: wavelength m
    assert abs(z[0] - np.sin(t / m)) < 1e-13 and abs(z[1] - np.cos(t / m)) < 1e-13
    ts = 1e-5
    zs = O.model_temporal_encoding(cfg, blob, ts)
    omega = np.arctan2(zs[0::2], zs[1::2]) / ts
    assert np.allclose(omega[1:] / omega[:-1], (5 * M / m) ** (-2.0 / d), rtol=1e-6)


def _torch_linear(cfg, blob, name_w, name_b, u):
    return Fn.linear(torch.as_tensor(u), torch.as_tensor(_get(cfg, blob, name_w)),
                     torch.as_tensor(_get(cfg, blob, name_b))).numpy()


def _h0(cfg, blob, tau, mk):
    t = np.cumsum(tau.astype(np.float64), axis=1)
    z = np.stack([[O.model_temporal_encoding(cfg, blob, x) for x in row] for row in t])
    return z, z + _get(cfg, blob, "type_emb")[mk]


def test_attnhp_zero_values_leave_the_embedding():
    blob = IN.model_blob(ATT_T, 2, 0, head_gain=3.0)
    d = ATT_T.d_model
    for l in range(ATT_T.layers):
        w = _get(ATT_T, blob, f"layer{l}.w_qkv").copy()
        w[2 * d:] = 0.0
        blob = _set(ATT_T, blob, f"layer{l}.w_qkv", w)
        b = _get(ATT_T, blob, f"layer{l}.b_qkv").copy()
        b[2 * d:] = 0.0
        blob = _set(ATT_T, blob, f"layer{l}.b_qkv", b)
    tau, mk = _hist(2, 15, 3, 4)
    _, h0 = _h0(ATT_T, blob, tau, mk)
    hd = O.score(ATT_T, blob, tau, mk)[0]
    assert np.abs(hd[:, :-1] - HP.torch_heads(ATT_T, blob, h0)[:, :-1]).max() < 1e-12


def test_attnhp_uniform_scores_give_the_damped_causal_mean():
    """Zero query / key weights: every f = 1, so a_i = sum_{j<=i} v_j / (i + 2)
    (i + 1 keys plus the 1 of the normaliser); h_1 = h_0 + tanh(a)."""
    cfg = CF.ModelCfg(1, 32, 2, 64, 4, 3, CF.FP32, CF.ATTNHP)
    blob = IN.model_blob(cfg, 6, 0, head_gain=3.0)
    d = cfg.d_model
    w = _get(cfg, blob, "layer0.w_qkv").copy()
    w[:2 * d] = 0.0
    b = _get(cfg, blob, "layer0.b_qkv").copy()
    b[:2 * d] = 0.0
    b[2 * d:] = np.linspace(-1.0, 1.0, d)
    blob = _set(cfg, _set(cfg, blob, "layer0.w_qkv", w), "layer0.b_qkv", b)
    tau, mk = _hist(2, 12, 3, 7)
    z, h0 = _h0(cfg, blob, tau, mk)
    u = np.concatenate([z, h0], -1)
    v = _torch_linear(cfg, blob, "layer0.w_qkv", "layer0.b_qkv", u)[..., 2 * d:]
    n = tau.shape[1]
    a = np.cumsum(v, axis=1) / (np.arange(n)[None, :, None] + 2.0)
    h1 = h0 + np.tanh(a)
    hd = O.score(cfg, blob, tau, mk)[0]
    assert np.abs(hd[:, :-1] - HP.torch_heads(cfg, blob, h1)[:, :-1]).max() < 1e-12


def test_attnhp_single_event_is_a_sigmoid_gate():
    """One event: a = e^s v / (1 + e^s) = sigmoid(s) v with
    s = q k / sqrt(d_head) per head; the head after it is head(h_0 + tanh(a))."""
    cfg = CF.ModelCfg(1, 32, 2, 64, 4, 3, CF.FP32, CF.ATTNHP)
    blob = IN.model_blob(cfg, 8, 0, head_gain=3.0)
    blob = _set(cfg, blob, "layer0.w_qkv", _get(cfg, blob, "layer0.w_qkv") * 40.0)
    d, nh = cfg.d_model, cfg.heads
    dh = d // nh
    tau, mk = _hist(4, 2, 3, 9)
    z, h0 = _h0(cfg, blob, tau, mk)
    u = np.concatenate([z, h0], -1)[:, 0]
    qkv = _torch_linear(cfg, blob, "layer0.w_qkv", "layer0.b_qkv", u)
    q, k, v = qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:]
    a = np.concatenate([torch.sigmoid(torch.as_tensor(
        (q[:, i * dh:(i + 1) * dh] * k[:, i * dh:(i + 1) * dh]).sum(1, keepdims=True) / np.sqrt(dh))).numpy()
        * v[:, i * dh:(i + 1) * dh] for i in range(nh)], 1)
    s_abs = np.abs((q * k).sum(1))
    assert s_abs.max() > 0.5                  # the gate is not near 1/2 everywhere
    hd = O.score(cfg, blob, tau, mk)[0]
    assert np.abs(hd[:, 0] - HP.torch_heads(cfg, blob, h0[:, 0] + np.tanh(a))).max() < 1e-12


def test_attnhp_cached_equals_recomputed_and_sampling_runs():
    blob_t = IN.model_blob(ATT_T, 3, 0, head_gain=2.0)
    dcfg = CF.ModelCfg(1, 16, 1, 32, 4, 3, CF.FP32, CF.ATTNHP)
    blob_d = IN.model_blob(dcfg, 3, 1, head_gain=2.0)
    tau, mk = _hist(3, 6, 3, 2)
    a = O.sample_sd(ATT_T, blob_t, dcfg, blob_d, tau, mk, 25, 4, seed=5)
    b = O.sample_sd(ATT_T, blob_t, dcfg, blob_d, tau, mk, 25, 4, seed=5, recompute=True)
    assert np.allclose(a["tau"], b["tau"], rtol=1e-9) and np.array_equal(a["k"], b["k"])
    ar = O.sample_ar(ATT_T, blob_t, tau, mk, 25, seed=5)
    same = O.sample_sd(ATT_T, blob_t, ATT_T, blob_t, tau, mk, 25, 4, seed=5)
    assert np.array_equal(ar["k"], same["k"]) and np.array_equal(ar["tau"], same["tau"])
