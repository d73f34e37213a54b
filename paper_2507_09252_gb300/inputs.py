"""Seeded synthetic inputs: model weight blobs and event histories.

This module is shared by the CUDA path, the oracle and the benchmark.  It
holds no arithmetic of the sampling method: it only draws random numbers and
lays them out in the weight-blob format that ``include/tppsd.h`` documents.

Weight recipe (random init standing in for the paper's trained models,
App. C.2): every matrix and the type embedding ~ N(0, 0.02); all biases 0;
LayerNorm gain 1, shift 0.  Target and draft are drawn from independent
streams.  bf16 models have each fp32 draw rounded once to bf16
(round-to-nearest-even) and stored back as fp32, so both sides read the same
exactly-representable values.

History recipes (stand-ins for the paper's datasets, App. B):
- "exp":            tau ~ Exp(rate), K = 1 mark
- "hawkes5":        5-D Hawkes, mu_k, alpha_kj = alpha for all k,j,
                    exponential kernel beta, simulated by Ogata thinning
                    (Sec. 2.2), mark drawn in proportion to lambda_k
- "gamma":          tau ~ Gamma(shape, scale), uniform marks
- "lognormal_zipf": tau ~ LogNormal(m, s), marks Zipf(a) truncated to 1..K
- "exp_uniform":    tau ~ Exp(rate), uniform marks
Inter-arrival times are clamped below at 1e-12 so that t is strictly
increasing.
"""
import numpy as np

from .configs import ModelCfg, Workload

INIT_STD = 0.02
TAU_MIN = 1e-12


# AttNHP temporal-encoding time scales (m, M) written into its blobs: the
# wavelengths of the encoding run from m to 5M.
ATTNHP_SCALES = (0.1, 1000.0)


def blob_layout(cfg: ModelCfg):
    """Ordered (name, shape, init) triples of the weight blob.

    init: "w" = N(0, 0.02), "0" = zeros, "1" = ones, "scales" = the AttNHP
    time scales above.  Matrices are row-major [out][in] (y = W x + b).
    THP and SAHP layers: QKV, output projection, two LayerNorms, FFN.
    AttNHP layers: QKV from [z(t); h] (2d inputs) only.  SAHP appends its
    per-dimension temporal frequencies, AttNHP its two time scales.
    """
    d, F, M, K = cfg.d_model, cfg.d_ffn, cfg.n_mix, cfg.n_marks
    enc = getattr(cfg, "encoder", 0)
    out = [("type_emb", (K, d), "w")]
    for l in range(cfg.layers):
        p = f"layer{l}."
        if enc == 2:
            out += [(p + "w_qkv", (3 * d, 2 * d), "w"), (p + "b_qkv", (3 * d,), "0")]
            continue
        out += [
            (p + "w_qkv", (3 * d, d), "w"), (p + "b_qkv", (3 * d,), "0"),
            (p + "w_o", (d, d), "w"), (p + "b_o", (d,), "0"),
            (p + "ln1_g", (d,), "1"), (p + "ln1_b", (d,), "0"),
            (p + "w_1", (F, d), "w"), (p + "b_1", (F,), "0"),
            (p + "w_2", (d, F), "w"), (p + "b_2", (d,), "0"),
            (p + "ln2_g", (d,), "1"), (p + "ln2_b", (d,), "0"),
        ]
    out += [
        ("head.E", (3 * d, d), "w"),
        ("head.v_w", (M, d), "w"), ("head.b_w", (M,), "0"),
        ("head.v_mu", (M, d), "w"), ("head.b_mu", (M,), "0"),
        ("head.v_s", (M, d), "w"), ("head.b_s", (M,), "0"),
        ("head.v_k1", (d, d), "w"), ("head.b_k1", (d,), "0"),
        ("head.v_k2", (K, d), "w"), ("head.b_k2", (K,), "0"),
    ]
    if enc == 1:
        out += [("tenc_w", (d,), "w")]
    elif enc == 2:
        out += [("tenc_scales", (2,), "scales")]
    return out


def blob_size(cfg: ModelCfg) -> int:
    return int(sum(np.prod(s) for _, s, _ in blob_layout(cfg)))


def blob_offsets(cfg: ModelCfg):
    """name -> (offset, shape) in floats."""
    off, table = 0, {}
    for name, shape, _ in blob_layout(cfg):
        table[name] = (off, shape)
        off += int(np.prod(shape))
    return table


def round_bf16(x: np.ndarray) -> np.ndarray:
    """fp32 -> nearest bf16 (ties to even), returned as fp32."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    b = (b + 0x7FFF + ((b >> 16) & 1)) & 0xFFFF0000
    return b.astype(np.uint32).view(np.float32)


def model_blob(cfg: ModelCfg, seed: int, role: int, head_gain: float = 1.0) -> np.ndarray:
    """Random-init weights for one model; role 0 = target, 1 = draft.

    ``head_gain`` scales the std of the head matrices (names "head.*"); the
    workloads use 1.  Tests use a larger gain so that the heads vary
    strongly from position to position.
    """
    rng = np.random.default_rng([seed, 7919, role, cfg.d_model, cfg.layers])
    parts = []
    for name, shape, init in blob_layout(cfg):
        n = int(np.prod(shape))
        if init == "w":
            std = INIT_STD * (head_gain if name.startswith("head.") else 1.0)
            parts.append(rng.normal(0.0, std, n).astype(np.float32))
        elif init == "1":
            parts.append(np.ones(n, np.float32))
        elif init == "scales":
            parts.append(np.array(ATTNHP_SCALES, np.float32))
        else:
            parts.append(np.zeros(n, np.float32))
    blob = np.concatenate(parts)
    if cfg.dtype == 1:
        blob = round_bf16(blob)
    return np.ascontiguousarray(blob, dtype=np.float32)


def shift_blob(cfg: ModelCfg, blob: np.ndarray, **deltas) -> np.ndarray:
    """Copy of ``blob`` with constants added to named bias vectors.

    Used to build draft models that differ from the target on purpose
    (e.g. ``shift_blob(cfg, b, **{"head.b_mu": 0.5})``).  A delta may be a
    scalar or an array of the vector's length.
    """
    out = blob.copy()
    offs = blob_offsets(cfg)
    for name, delta in deltas.items():
        o, shape = offs[name]
        n = int(np.prod(shape))
        out[o:o + n] += np.asarray(delta, dtype=np.float32)
    if cfg.dtype == 1:
        out = round_bf16(out)
    return out


def _hawkes5(rng, n, mu, alpha, beta, K=5):
    """Ogata thinning for a K-dim Hawkes process with all alpha_kj equal."""
    taus = np.empty(n, np.float64)
    marks = np.empty(n, np.int32)
    t, last_t, excite = 0.0, 0.0, 0.0  # excite = sum_i exp(-beta (t - t_i))
    i = 0
    while i < n:
        lam_bar = K * (mu + alpha * excite)        # intensity only decays
        t_new = t + rng.exponential(1.0 / lam_bar)
        excite *= np.exp(-beta * (t_new - t))
        t = t_new
        lam_k = mu + alpha * excite                 # same for every k
        if rng.uniform() * lam_bar < K * lam_k:
            taus[i] = t - last_t
            marks[i] = rng.integers(0, K)           # proportional to equal lambda_k
            last_t = t
            excite += 1.0
            i += 1
    return taus, marks


def histories(w: Workload, batch: int = None, seed: int = None):
    """(tau [B][H] float32, marks [B][H] int32) for workload ``w``."""
    B = w.batch if batch is None else batch
    H = w.hist_len
    K = w.target.n_marks
    seed = w.seed if seed is None else seed
    rng = np.random.default_rng([seed, 104729, B, H])
    kind, p = w.history.kind, w.history.params
    if kind == "exp":
        tau = rng.exponential(1.0 / p[0], (B, H))
        marks = np.zeros((B, H), np.int32)
    elif kind == "exp_uniform":
        tau = rng.exponential(1.0 / p[0], (B, H))
        marks = rng.integers(0, K, (B, H)).astype(np.int32)
    elif kind == "gamma":
        tau = rng.gamma(p[0], p[1], (B, H))
        marks = rng.integers(0, K, (B, H)).astype(np.int32)
    elif kind == "lognormal_zipf":
        tau = rng.lognormal(p[0], p[1], (B, H))
        pk = np.arange(1, K + 1, dtype=np.float64) ** (-p[2])
        marks = rng.choice(K, size=(B, H), p=pk / pk.sum()).astype(np.int32)
    elif kind == "hawkes5":
        tau = np.empty((B, H))
        marks = np.empty((B, H), np.int32)
        for b in range(B):
            tau[b], marks[b] = _hawkes5(rng, H, p[0], p[1], p[2], K)
    else:
        raise ValueError(kind)
    tau = np.maximum(tau, TAU_MIN).astype(np.float32)
    return np.ascontiguousarray(tau), np.ascontiguousarray(marks)


def workload_inputs(w: Workload, batch: int = None):
    """Blobs and histories of a workload: (blob_T, blob_D, tau, marks)."""
    bt = model_blob(w.target, w.seed, 0)
    bd = model_blob(w.draft, w.seed, 1)
    tau, marks = histories(w, batch)
    return bt, bd, tau, marks
