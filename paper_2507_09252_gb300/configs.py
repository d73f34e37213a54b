"""Workload definitions: model shapes and synthetic-input recipes.

Five workloads, shaped like the paper's experiments (Sec. 5.2-5.4, App. C):
a tiny fp32 univariate model, the Hawkes-history headline shape, a K=22
gamma sweep (Fig. 3 shape), a long-context K=50 model, and a batch x draft
size sweep (Tab. 3 shape).  Weights are random-init N(0, 0.02); the paper's
trained weights and datasets are not available, so these synthetic inputs
stand in for them.

Every field the paper leaves open is fixed here:
- mark-head hidden width = d_model (Sec. 4.2 leaves the width of V_k^(1) open);
- draft FFN = 4*d_draft, except the tiny fp32 workload (2*d = 32);
- draft heads: d32 -> 2, d64 -> 4, d128 -> 4;
- sweep workload: M = 8, target FFN 1024.
"""
from dataclasses import dataclass, field, replace
from typing import Tuple

FP32 = 0
BF16 = 1
THP, SAHP, ATTNHP = 0, 1, 2  # history encoders of App. D.4


@dataclass(frozen=True)
class ModelCfg:
    layers: int
    d_model: int
    heads: int
    d_ffn: int
    n_mix: int
    n_marks: int
    dtype: int  # FP32 or BF16
    encoder: int = 0  # THP, SAHP or ATTNHP (App. D.4)

    @property
    def d_head(self) -> int:
        return self.d_model // self.heads


@dataclass(frozen=True)
class History:
    kind: str            # "exp", "hawkes5", "gamma", "lognormal_zipf", "exp_uniform"
    params: Tuple = ()


@dataclass(frozen=True)
class Workload:
    name: str
    target: ModelCfg
    draft: ModelCfg
    batch: int
    hist_len: int
    n_events: int
    gamma: int
    history: History
    seed: int = 0
    gammas: Tuple[int, ...] = ()      # sweep values (workload 3)
    batches: Tuple[int, ...] = ()     # sweep values (workload 5)
    drafts: Tuple[ModelCfg, ...] = () # sweep values (workload 5)

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


def _m(layers, d, heads, ffn, mix, marks, dtype):
    return ModelCfg(layers, d, heads, ffn, mix, marks, dtype)


# 1: univariate K=1, fp32, tiny (the case the oracle finishes in seconds)
C1 = Workload(
    name="c1_univariate_fp32",
    target=_m(2, 32, 2, 64, 4, 1, FP32),
    draft=_m(1, 16, 1, 32, 4, 1, FP32),
    batch=4, hist_len=16, n_events=64, gamma=4,
    history=History("exp", (1.0,)),
)

# 2: K=5 Hawkes histories, bf16 (the headline throughput shape)
C2 = Workload(
    name="c2_hawkes_k5_bf16",
    target=_m(4, 128, 4, 512, 8, 5, BF16),
    draft=_m(1, 32, 2, 128, 8, 5, BF16),
    batch=256, hist_len=64, n_events=512, gamma=8,
    history=History("hawkes5", (0.2, 0.3, 1.0)),
)

# 3: K=22, Gamma(0.5, 2) histories, gamma sweep
C3 = Workload(
    name="c3_gamma_k22_bf16",
    target=_m(6, 256, 8, 1024, 8, 22, BF16),
    draft=_m(2, 64, 4, 256, 8, 22, BF16),
    batch=1024, hist_len=128, n_events=1024, gamma=8,
    history=History("gamma", (0.5, 2.0)),
    gammas=(2, 4, 8, 12, 16),
)

# 4: long sequences, K=50, LogNormal(0,1) times + Zipf(1.1) marks
C4 = Workload(
    name="c4_long_k50_bf16",
    target=_m(8, 512, 8, 2048, 16, 50, BF16),
    draft=_m(2, 128, 4, 512, 16, 50, BF16),
    batch=64, hist_len=512, n_events=4096, gamma=10,
    history=History("lognormal_zipf", (0.0, 1.0, 1.1)),
)

_C5_DRAFTS = (
    _m(1, 32, 2, 128, 8, 100, BF16),
    _m(2, 64, 4, 256, 8, 100, BF16),
    _m(2, 128, 4, 512, 8, 100, BF16),
)

# 5: batch x draft-size sweep, K=100
C5 = Workload(
    name="c5_sweep_k100_bf16",
    target=_m(6, 256, 8, 1024, 8, 100, BF16),
    draft=_C5_DRAFTS[1],
    batch=256, hist_len=64, n_events=256, gamma=8,
    history=History("exp_uniform", (1.0,)),
    batches=(1, 16, 256, 4096),
    drafts=_C5_DRAFTS,
)

WORKLOADS = {w.name: w for w in (C1, C2, C3, C4, C5)}
BY_INDEX = [C1, C2, C3, C4, C5]
