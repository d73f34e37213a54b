"""Multi-rank logic of bench.py on CPU: two gloo ranks, each with its own
independent batch, whole-job time = the slowest rank's, whole-job rate =
all ranks' events over that time."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    from paper_2507_09252_gb300 import configs as CF
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        wl = CF.C1
        tau, mk = bench.rank_histories(wl, rank)
        ms = 10.0 + 5.0 * rank                # rank 1 is the slow one
        job_ms = bench.max_over_ranks(ms, world, "cpu")
        q.put((rank, job_ms, bench.job_rate(world, wl.batch, wl.n_events, job_ms),
               tau.tobytes(), mk.tobytes()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in range(2)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res.sort()
    sys.path.insert(0, ROOT)
    from paper_2507_09252_gb300 import configs as CF
    wl = CF.C1
    for _, job_ms, rate, _, _ in res:
        assert job_ms == pytest.approx(15.0)
        assert rate == pytest.approx(2 * wl.batch * wl.n_events / 0.015)
    # each rank's histories are its own (no shared units)
    assert res[0][3] != res[1][3]


def test_single_rank_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5, 1, "cpu") == 3.5
    assert bench.job_rate(1, 256, 512, 1000.0) == pytest.approx(256 * 512)
    from paper_2507_09252_gb300 import configs as CF
    a = bench.rank_histories(CF.C1, 0)
    b = bench.rank_histories(CF.C1, 0)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_traffic_record_is_dropped_when_a_source_changes(tmp_path, monkeypatch):
    """bench.py reports an ncu DRAM figure only while every source file the
    capture was taken on is byte-identical."""
    import hashlib
    import json
    sys.path.insert(0, ROOT)
    import bench
    (tmp_path / "profiles").mkdir()
    src = tmp_path / "k.cu"
    src.write_text("kernel v1")
    rec = {"kernels": {"draft": {"dram_bytes_per_launch": 123,
                                 "sources": {"k.cu": hashlib.sha256(b"kernel v1").hexdigest()}}}}
    (tmp_path / "profiles" / "dram_traffic_c2.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.ncu_traffic("draft") == 123
    assert bench.ncu_traffic("attention") is None
    src.write_text("kernel v2")
    assert bench.ncu_traffic("draft") is None


def test_roofline_reports_every_class():
    """bench.py's roofline: the dominant class (largest device time) with
    its algorithmic figure, and every class's own fraction; the fused
    post-attention block counts O-proj + FFN1 + FFN2 FLOPs."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2507_09252_gb300 import configs as CF
    kt = {"draft": (7.0, 70), "attention": (5.5, 280), "gemm_ffn2": (4.7, 280), "gemm_qkv": (2.8, 280),
          "head": (1.4, 70), "epilogue": (1.1, 70), "control": (0.4, 70), "gemm_o": (0.0, 0)}
    stats = {"rounds": 16376, "drafted": 131008, "accepted": 115668, "target_keys": 5340083}
    peaks = {"hbm_gbs": 6682.5, "bf16_tflops_sustained": 1772.7}
    dom, per = bench.roofline(kt, stats, CF.C2, peaks)
    assert dom["kernel"] == "draft" and dom["unit"] == "GB/s" and 0 < dom["frac"] < 1
    assert set(per) == {k for k, v in kt.items() if v[1]}
    T = CF.C2.target
    rows = stats["rounds"] * (CF.C2.gamma + 1)
    flops = 2.0 * rows * (T.d_model ** 2 + 2 * T.d_model * T.d_ffn) * T.layers / 280
    assert per["gemm_ffn2"]["bound"] == "tensor"
    assert per["gemm_ffn2"]["achieved"] == pytest.approx(flops / (4.7e-3 / 280) / 1e12, rel=1e-3)
    assert per["control"]["bound"] == "latency"
    assert abs(sum(v["share_of_device_time"] for v in per.values()) - 1.0) < 0.01
