"""Roofline arithmetic of bench.py on CPU, fed with the per-class CUDA-event
totals and counters of one recorded headline call (256 sequences, 512
events, gamma = 8, 70 rounds): the dominant class is the one with the
largest device time, every class's algorithmic rate stays below the copy
peak, and the per-launch units are the ones the formulas state."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2507_09252_gb300 import configs as CF  # noqa: E402

KT = {"draft": (3.965, 70), "embed": (0.611, 70), "gemm_qkv": (2.402, 280), "attention": (5.167, 280),
      "gemm_o": (0.0, 0), "gemm_ffn2": (4.693, 280), "head": (0.948, 70), "epilogue": (1.152, 70),
      "control": (0.428, 70), "begin": (0.004, 1)}
STATS = {"rounds": 16375, "drafted": 131000, "accepted": 115666, "emitted": 132041,
         "resample_iters": 115012, "cap_hits": 0, "loop_iters": 70, "target_keys": 5339489,
         "draft_keys": 46230265}
PEAKS = {"hbm_gbs": 6682.5, "bf16_tflops_sustained": 1772.7}


def test_dominant_class_and_bounds():
    dom, per = bench.roofline(KT, STATS, CF.C2, PEAKS)
    assert dom["kernel"] == "attention" and dom["bound"] == "hbm" and dom["unit"] == "GB/s"
    assert set(per) == {k for k, v in KT.items() if v[1] > 0}
    assert abs(sum(v["share_of_device_time"] for v in per.values()) - 1.0) < 0.01
    for name, r in per.items():
        assert 0.0 < r["frac"] < 1.0, (name, r)


def test_per_launch_units():
    wl = CF.C2
    T = wl.target
    d, F, L = T.d_model, T.d_ffn, T.layers
    rows = STATS["rounds"] * (wl.gamma + 1)
    _, per = bench.roofline(KT, STATS, wl, PEAKS)
    # attention: K and V of every attended key once per (sequence, layer) + Q and output rows
    att = (STATS["target_keys"] + rows) * L * 2 * d * 2 / 280
    assert per["attention"]["achieved"] == pytest.approx(att / (5.167e-3 / 280) / 1e9, rel=1e-3)
    assert 30e6 < att < 50e6
    # QKV: 2 R (3d) d flops per launch; the fused block: 2 R (d^2 + 2 d F)
    qkv = 2.0 * rows * 3 * d * d * L / 280
    assert per["gemm_qkv"]["achieved"] == pytest.approx(qkv / (2.402e-3 / 280) / 1e12, rel=1e-3)
    ffn = 2.0 * rows * (d * d + 2 * d * F) * L / 280
    assert per["gemm_ffn2"]["achieved"] == pytest.approx(ffn / (4.693e-3 / 280) / 1e12, rel=1e-3)
    # begin: one launch initialising B x N output events (16 bytes each)
    assert per["begin"]["achieved"] == pytest.approx(wl.batch * wl.n_events * 16 / 4e-6 / 1e9, rel=1e-3)


def test_path_roofline():
    """The whole path's ideal time is the sum of the classes' ideal times
    and is a small fraction of the recorded 15.30 ms step."""
    _, per = bench.roofline(KT, STATS, CF.C2, PEAKS)
    pr = bench.path_roofline(per, 15.30)
    parts = sum(r["algorithmic_per_launch"] * r["launches"] / (r["peak"] * (1e12 if r["unit"] == "TFLOP/s" else 1e9))
                for r in per.values())
    assert pr["ideal_ms"] == pytest.approx(parts * 1e3, abs=1e-3)
    assert 0.05 < pr["frac"] < 0.3
    att = per["attention"]
    assert att["algorithmic_per_launch"] * 280 / (att["peak"] * 1e9) * 1e3 > 0.5 * pr["ideal_ms"]


def test_bench_calls_attention_figure_and_length_overrides():
    """bench_calls' attention figure is bench.py's attention class (one
    formula), and --hist-len / --n-events reshape the workload so that a
    long history puts every round's context past that many keys."""
    import bench_calls
    r = bench_calls.attention_roofline(5.167, 280, STATS, CF.C2)
    _, per = bench.roofline(KT, STATS, CF.C2, {"hbm_gbs": bench_calls._hbm_peak(), "bf16_tflops_sustained": 1772.7})
    assert r["achieved_GBps"] == pytest.approx(per["attention"]["achieved"], rel=1e-6)
    assert r["bytes_per_launch"] == int(per["attention"]["algorithmic_per_launch"])
    assert r["mean_keys_per_sequence"] == pytest.approx(STATS["target_keys"] / STATS["rounds"], abs=0.05)
    wl = CF.C4.with_(hist_len=4096, n_events=256)
    assert (wl.hist_len, wl.n_events, wl.batch, wl.gamma) == (4096, 256, CF.C4.batch, CF.C4.gamma)
