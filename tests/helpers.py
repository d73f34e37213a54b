"""Shared test helpers: random heads, closed-form mixture CDF, model pins.

The closed forms here come from the mathematics (log-normal CDF via the
normal CDF, Sec. 4.2 / App. A.1) and from library routines (scipy, torch);
none of them calls the oracle.
"""
import numpy as np
from scipy import stats


def random_head(rng, M, K, mu_scale=0.7, s_scale=0.4, w_scale=1.0, k_scale=1.0):
    """A head row [log w | mu | s | log f] with normalised log w and log f."""
    lw = rng.normal(0, w_scale, M)
    lw -= np.log(np.exp(lw).sum())
    mu = rng.normal(0, mu_scale, M)
    s = rng.normal(0, s_scale, M)
    lf = rng.normal(0, k_scale, K)
    lf -= np.log(np.exp(lf).sum())
    return np.concatenate([lw, mu, s, lf])


def mixture_cdf(head, M, tau):
    """G(tau) = sum_m w_m Phi((log tau - mu_m) / sigma_m)."""
    w = np.exp(head[:M]); mu = head[M:2 * M]; sig = np.exp(head[2 * M:3 * M])
    lt = np.log(np.asarray(tau, dtype=np.float64))[..., None]
    return (w * stats.norm.cdf((lt - mu) / sig)).sum(-1)


def mixture_pdf(head, M, tau):
    """g(tau) from scipy's log-normal pdf (library routine)."""
    w = np.exp(head[:M]); mu = head[M:2 * M]; sig = np.exp(head[2 * M:3 * M])
    tau = np.asarray(tau, dtype=np.float64)
    return sum(w[m] * stats.lognorm.pdf(tau, s=sig[m], scale=np.exp(mu[m])) for m in range(M))


def residual_cdf_factory(head_t, head_d, M, grid_lo=-12.0, grid_hi=12.0, n=200001):
    """CDF of g' = max(0, g_T - g_D) / Z, by quadrature on a log-tau grid."""
    x = np.linspace(grid_lo, grid_hi, n)
    tau = np.exp(x)
    r = np.maximum(0.0, mixture_pdf(head_t, M, tau) - mixture_pdf(head_d, M, tau)) * tau
    c = np.concatenate([[0.0], np.cumsum(0.5 * (r[1:] + r[:-1]) * np.diff(x))])
    Z = c[-1]
    return (lambda t: np.interp(np.log(t), x, c / Z)), Z


def chi2_pvalue(observed, expected):
    observed = np.asarray(observed, float)
    expected = np.asarray(expected, float)
    keep = expected > 0
    stat = (((observed - expected) ** 2)[keep] / expected[keep]).sum()
    dof = keep.sum() - 1
    return stats.chi2.sf(stat, dof)


def torch_heads(cfg, blob, x):
    """Heads of Sec. 4.2 on hidden states x [..., d] with F.linear and
    log_softmax in float64: [..., 3M+K] = [log w | mu | log sigma | log f]."""
    import torch
    import torch.nn.functional as Fn
    from paper_2507_09252_gb300.inputs import blob_offsets

    offs = blob_offsets(cfg)
    bt = torch.from_numpy(np.asarray(blob, np.float64))

    def P(name):
        o, shape = offs[name]
        return bt[o:o + int(np.prod(shape))].reshape(shape)

    d = cfg.d_model
    x = torch.as_tensor(np.asarray(x, np.float64))
    with torch.no_grad():
        e = Fn.linear(x, P("head.E"))
        lw = torch.log_softmax(Fn.linear(e[..., :d], P("head.v_w"), P("head.b_w")), -1)
        mu = Fn.linear(e[..., d:2 * d], P("head.v_mu"), P("head.b_mu"))
        s = Fn.linear(e[..., 2 * d:], P("head.v_s"), P("head.b_s"))
        a = torch.tanh(Fn.linear(x, P("head.v_k1"), P("head.b_k1")))
        lf = torch.log_softmax(Fn.linear(a, P("head.v_k2"), P("head.b_k2")), -1)
    return torch.cat([lw, mu, s, lf], -1).numpy()


def torch_reference_heads(cfg, blob, tau, marks, z=None):
    """Heads of one model built from torch library modules in float64.

    The encoder is torch.nn.TransformerEncoderLayer (post-LN, ReLU, eps 1e-5,
    causal mask); the temporal encoding and heads use torch.sin/cos,
    F.linear and log_softmax.  Returns [B][n][3M+K] (row i = head after
    events 0..i).  z [B][n][d], if given, replaces the THP temporal
    encoding (for encoders whose encoding is pinned separately).
    """
    import torch
    import torch.nn.functional as Fn
    from paper_2507_09252_gb300.inputs import blob_offsets

    offs = blob_offsets(cfg)
    bt = torch.from_numpy(np.asarray(blob, np.float64))

    def P(name):
        o, shape = offs[name]
        n = int(np.prod(shape))
        return bt[o:o + n].reshape(shape)

    d, M = cfg.d_model, cfg.n_mix
    layers = []
    for l in range(cfg.layers):
        lay = torch.nn.TransformerEncoderLayer(d, cfg.heads, cfg.d_ffn, dropout=0.0,
                                               activation="relu", layer_norm_eps=1e-5,
                                               batch_first=True, norm_first=False,
                                               dtype=torch.float64)
        with torch.no_grad():
            p = f"layer{l}."
            lay.self_attn.in_proj_weight.copy_(P(p + "w_qkv"))
            lay.self_attn.in_proj_bias.copy_(P(p + "b_qkv"))
            lay.self_attn.out_proj.weight.copy_(P(p + "w_o"))
            lay.self_attn.out_proj.bias.copy_(P(p + "b_o"))
            lay.norm1.weight.copy_(P(p + "ln1_g")); lay.norm1.bias.copy_(P(p + "ln1_b"))
            lay.linear1.weight.copy_(P(p + "w_1")); lay.linear1.bias.copy_(P(p + "b_1"))
            lay.linear2.weight.copy_(P(p + "w_2")); lay.linear2.bias.copy_(P(p + "b_2"))
            lay.norm2.weight.copy_(P(p + "ln2_g")); lay.norm2.bias.copy_(P(p + "ln2_b"))
        lay.eval()
        layers.append(lay)
    tau = torch.from_numpy(np.asarray(tau, np.float64))
    t = torch.cumsum(tau, dim=1)
    B, n = t.shape
    j = torch.arange(d, dtype=torch.float64)
    je = j - (j.long() % 2).double()
    arg = t[..., None] / torch.pow(torch.tensor(10000.0, dtype=torch.float64), je / d)
    if z is None:
        z = torch.where((j.long() % 2) == 1, torch.cos(arg), torch.sin(arg))
    else:
        z = torch.as_tensor(np.asarray(z, np.float64))
    x = z + P("type_emb")[torch.from_numpy(np.asarray(marks, np.int64))]
    mask = torch.triu(torch.full((n, n), float("-inf"), dtype=torch.float64), diagonal=1)
    with torch.no_grad():
        for lay in layers:
            x = lay(x, src_mask=mask)
        e = Fn.linear(x, P("head.E"))
        lw = torch.log_softmax(Fn.linear(e[..., :d], P("head.v_w"), P("head.b_w")), -1)
        mu = Fn.linear(e[..., d:2 * d], P("head.v_mu"), P("head.b_mu"))
        s = Fn.linear(e[..., 2 * d:], P("head.v_s"), P("head.b_s"))
        a = torch.tanh(Fn.linear(x, P("head.v_k1"), P("head.b_k1")))
        lf = torch.log_softmax(Fn.linear(a, P("head.v_k2"), P("head.b_k2")), -1)
    return torch.cat([lw, mu, s, lf], -1).numpy()


def pit_times(rows, M, taus):
    """u_i = G(tau_i | head_i): iid Uniform(0,1) when each tau_i is drawn from
    its head's mixture given the past (probability integral transform; the
    time-rescaling statistic of App. A.4 with the model as ground truth)."""
    w = np.exp(rows[:, :M]); mu = rows[:, M:2 * M]; sg = np.exp(rows[:, 2 * M:3 * M])
    lt = np.log(np.asarray(taus, np.float64))[:, None]
    return (w * stats.norm.cdf((lt - mu) / sg)).sum(1)


def pit_marks(rows, M, ks, rng):
    """Randomised PIT of discrete marks: F(k-1) + V f(k), V ~ U(0,1), is iid
    Uniform(0,1) when each k_i is drawn from its head's f given the past."""
    f = np.exp(rows[:, 3 * M:])
    f = f / f.sum(1, keepdims=True)
    cdf_below = np.cumsum(f, 1) - f
    idx = np.arange(len(ks))
    return cdf_below[idx, ks] + rng.uniform(size=len(ks)) * f[idx, ks]
