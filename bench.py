"""Benchmark of the TPP-SD sampler on the headline workload.

Workload: target 4 layers d128 4 heads FFN 512, draft 1 layer d32 2 heads,
8-component log-normal mixture, K=5 marks, bf16 weights with fp32
accumulation; 256 sequences with 64-event Hawkes histories, 512 new events
each, gamma = 8.  Random-init weights and seeded synthetic histories.

One step = prefill (encode the history with both models) + TPP-SD sampling
of all events, inputs resident in HBM.  Reported:
  value         sampled events/s over all ranks (device-timed steps)
  ar            the same for target-only autoregressive sampling
  e2e           events/s through the C ABI with pinned HOST buffers, the
                host->device history copy and device->host result copy
                inside the timed region
  roofline      the dominant kernel class (from a profiled call with CUDA
                events around every launch) against the measured peak
  cpu_baseline  the CPU oracle on a bounded sample of the same workload

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Multi-GPU: one process per GPU under torchrun; every rank samples its own
256 sequences (weak scaling, no data-path collective).
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2507_09252_gb300 import configs as CF  # noqa: E402
from paper_2507_09252_gb300 import inputs as IN  # noqa: E402

METRIC = "sampled events/sec/GPU, TPP-SD vs AR target-only; mean accepted per verify"
UNIT = "events/s"
L2_BYTES = 129 * 1024 * 1024


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--host-loop", action="store_true",
                    help="launch every round's kernels from the host instead of one CUDA graph "
                         "(same kernels; lets a per-launch profiler see them)")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def rank_histories(wl, rank):
    """Histories of one rank: every rank samples its own batch of
    independent sequences (seed offset by the rank), so nothing is exchanged
    on the data path."""
    return IN.histories(wl, seed=wl.seed + rank)


def max_over_ranks(ms, world, device):
    """Step time of the whole job: the slowest rank's (MAX all-reduce)."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(world, batch, n_events, ms):
    """Events per second over all ranks (weak scaling: batch per rank)."""
    return world * batch * n_events / (ms / 1e3)


def workload_config(wl, rank_seed):
    return {"workload": wl.name, "batch_per_gpu": wl.batch, "hist_len": wl.hist_len,
            "n_events": wl.n_events, "gamma": wl.gamma,
            "target": "4L d128 4h F512 M8 K5", "draft": "1L d32 2h F128 M8 K5",
            "history": "5-D Hawkes (mu 0.2, alpha 0.3, beta 1) by thinning",
            "weights": "random init N(0, 0.02)", "seed": rank_seed,
            "l2": "flushed between timed steps (256 MiB write)",
            "step": "prefill + sample"}


# ---------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples every 50 ms while the timed region runs."""
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index, self.proc, self.lines = index, None, []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0])); mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------- roofline
def class_roofline(name, ms, launches, stats, wl, peaks, fused):
    """Algorithmic bytes (or FLOPs) per launch of one kernel class of a
    profiled SD call ÷ its mean CUDA-event time, against the measured peak.

    attention:  K and V of every cached position read once per (sequence,
                layer) + Q read + output write:  target_keys * 2 d eb + 2 R d eb
    draft:      draft K/V of each sequence loaded once per round (the kernel
                keeps it in shared memory for the round) + draft heads
                written + the draft model once per launch (L2-resident)
    gemm_*:     2 R N K FLOPs per layer (tcgen05 bf16 path for bf16 models);
                the fused post-attention block (timed as gemm_ffn2) does
                2 R (d^2 + 2 d F)
    head:       h rows read + head rows written + head weights
    embed:      per verify row: (t, k) read, fp32 and storage-type rows written
    epilogue:   per (sequence, round): target heads of gamma+1 rows and draft
                heads of gamma rows read, up to gamma+1 events written
    control:    n_emit and done of every sequence read
    begin:      the output arrays initialised (tau, t, k of B x N events)
    The last four are latency-bound; their figures say how far they are
    from moving bytes at all.
    """
    T, D = wl.target, wl.draft
    eb = 2 if T.dtype == CF.BF16 else 4
    rounds = stats["rounds"]                         # (sequence, round) pairs
    rows = rounds * (wl.gamma + 1)                   # verify rows over the call
    d, F, L = T.d_model, T.d_ffn, T.layers
    W = 3 * T.n_mix + T.n_marks
    per_launch_s = ms / 1e3 / max(launches, 1)
    bound, unit = "hbm", "GB/s"
    if name == "attention":
        total = stats["target_keys"] * L * 2 * d * eb + rows * L * 2 * d * eb
    elif name == "draft":
        from paper_2507_09252_gb300.tppsd import tppsd_blob_floats
        wbytes = tppsd_blob_floats(D) * 4
        # target_keys = sum over (sequence, round) of the context the round
        # attends, i.e. the draft KV positions the round loads once
        total = (stats["target_keys"] * D.layers * 2 * D.d_model * eb
                 + launches * wbytes + stats["drafted"] * (3 * D.n_mix + D.n_marks) * 4)
    elif name == "head":
        total = rows * (d + W) * 4 + launches * (4 * d * d + (3 * T.n_mix + T.n_marks + d) * d) * 4
    elif name.startswith("gemm"):
        nk = {"gemm_qkv": (3 * d, d), "gemm_o": (d, d), "gemm_ffn1": (F, d), "gemm_ffn2": (d, F)}[name]
        total = 2.0 * rows * nk[0] * nk[1] * L
        if name == "gemm_ffn2" and fused:
            total = 2.0 * rows * (d * d + 2 * d * F) * L
        bound, unit = "tensor", "TFLOP/s"
    else:
        if name == "embed":
            total = rows * (12 + d * (4 + eb))
        elif name == "epilogue":
            total = rounds * ((2 * wl.gamma + 1) * W * 4 + (wl.gamma + 1) * 16)
        elif name == "control":
            total = launches * wl.batch * 8
        elif name == "begin":
            total = launches * wl.batch * wl.n_events * 16
        else:
            total = rows * d * 4 * 2
        bound = "latency"
    per_launch = total / max(launches, 1)
    if bound == "tensor":
        achieved = per_launch / per_launch_s / 1e12
        # dense bf16 tensor peak, sustained (the kernel runs inside a long step)
        peak = peaks.get("bf16_tflops_sustained", 1700.0)
    else:
        achieved = per_launch / per_launch_s / 1e9
        peak = peaks.get("hbm_gbs", 6800.0)
    return {"bound": bound, "achieved": round(achieved, 2), "peak": round(peak, 1), "unit": unit,
            "frac": round(achieved / peak, 4), "per_launch_ms": round(per_launch_s * 1e3, 4),
            "launches": launches, "algorithmic_per_launch": per_launch}


def roofline(kt, stats, wl, peaks):
    """The dominant kernel class of a profiled SD call (largest share of the
    device time) with its roofline, plus every class's own figures."""
    fused = kt.get("gemm_o", (0.0, 0))[1] == 0 and kt.get("gemm_ffn2", (0.0, 0))[1] > 0
    live = {k: v for k, v in kt.items() if v[1] > 0}
    tot = sum(v[0] for v in live.values())
    per = {k: {**class_roofline(k, ms, n, stats, wl, peaks, fused), "share_of_device_time": round(ms / tot, 3)}
           for k, (ms, n) in live.items()}
    name = max(live, key=lambda k: live[k][0])
    top = per[name]
    dom = {"kernel": name, "bound": "hbm" if top["bound"] == "latency" else top["bound"],
           "achieved": top["achieved"], "peak": top["peak"], "unit": top["unit"], "frac": top["frac"],
           "traffic": ncu_traffic(name), "per_launch_ms": top["per_launch_ms"], "launches": top["launches"],
           "share_of_device_time": top["share_of_device_time"],
           "algorithmic_per_launch": top["algorithmic_per_launch"],
           "peak_source": "MEASURED_PEAKS.json" if peaks else "fallback"}
    return dom, per


def path_roofline(per, ms_step):
    """The whole path against its roofline: every kernel class's algorithmic
    bytes over the profiled call at the measured HBM peak (FLOPs at the
    tensor peak for the tensor-core classes), summed, over the measured step
    time (whose prefill the profiled call leaves out, so the fraction is a
    lower bound)."""
    ideal_s = 0.0
    for r in per.values():
        scale = 1e12 if r["unit"] == "TFLOP/s" else 1e9
        ideal_s += r["algorithmic_per_launch"] * r["launches"] / (r["peak"] * scale)
    return {"ideal_ms": round(ideal_s * 1e3, 3), "measured_ms": round(ms_step, 3),
            "frac": round(ideal_s * 1e3 / ms_step, 4)}


def ncu_traffic(kernel_class):
    """DRAM bytes per launch of a kernel class from the committed ncu capture
    (profiles/dram_traffic_c2.json), or None once any source file the
    capture was taken on has changed since."""
    import hashlib
    try:
        t = json.load(open(os.path.join(ROOT, "profiles", "dram_traffic_c2.json")))
        e = t["kernels"][kernel_class]
        for f, digest in e["sources"].items():
            with open(os.path.join(ROOT, f), "rb") as fh:
                if hashlib.sha256(fh.read()).hexdigest() != digest:
                    return None
        return e["dram_bytes_per_launch"]
    except (OSError, ValueError, KeyError):
        return None


def load_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except (OSError, ValueError):
        return {}


# ---------------------------------------------------------------- CPU oracle
def cpu_oracle_rate(wl, bt, bd, tau, mk, budget_s=12.0):
    """Oracle TPP-SD events/s on the first S sequences (S sized so that the
    run takes about budget_s), OpenMP over sequences on all host cores."""
    from oracle import oracle as O
    cores = os.cpu_count() or 1
    t0 = time.perf_counter()
    O.sample_sd(wl.target, bt, wl.draft, bd, tau[:1], mk[:1], wl.n_events, wl.gamma, 1, nthreads=1)
    one = time.perf_counter() - t0
    S = int(max(1, min(wl.batch, budget_s / max(one, 1e-3) * cores * 0.8)))
    S = max(cores, (S // cores) * cores) if S >= cores else S
    S = min(S, wl.batch)
    t0 = time.perf_counter()
    O.sample_sd(wl.target, bt, wl.draft, bd, tau[:S], mk[:S], wl.n_events, wl.gamma, 1, nthreads=cores)
    dt = time.perf_counter() - t0
    return {"value": round(S * wl.n_events / dt, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"first {S} of {wl.batch} sequences, all {wl.n_events} events, gamma "
                      f"{wl.gamma}, fp64 oracle with bf16 emulation, {dt:.1f} s",
            "value_1core": round(wl.n_events / max(one, 1e-9), 1)}


# ---------------------------------------------------------------- reference arm
def run_reference(args, wl):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    bt, bd, tau, mk = IN.workload_inputs(wl)
    from oracle import oracle as O
    cores = os.cpu_count() or 1
    S = min(wl.batch, 2 * cores)
    times = []
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        O.sample_sd(wl.target, bt, wl.draft, bd, tau[:S], mk[:S], wl.n_events, wl.gamma, 1,
                    nthreads=cores)
        if i >= args.warmup:
            times.append(time.perf_counter() - t0)
    ms = 1e3 * sum(times) / len(times)
    value = S * wl.n_events / (ms / 1e3)
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 1), "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(ms, 3), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {**workload_config(wl, wl.seed), "reference": "CPU oracle (fp64 C, bf16 emulation)",
                       "sample_sequences": S},
            "cpu_baseline": {"value": round(value, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"first {S} of {wl.batch} sequences per step"},
            "e2e": {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------- our arm
def main():
    args = parse()
    wl = CF.C2
    if args.impl == "reference":
        return run_reference(args, wl)
    import torch
    import torch.distributed as dist

    from paper_2507_09252_gb300 import tppsd as T
    from paper_2507_09252_gb300.sampler import Sampler, fit_poisson_draft

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", init_method="env://")
    B, H, N, g = wl.batch, wl.hist_len, wl.n_events, wl.gamma
    bt, bd = IN.model_blob(wl.target, wl.seed, 0), IN.model_blob(wl.draft, wl.seed, 1)
    tau_np, mk_np = rank_histories(wl, rank)
    s = Sampler(wl.target, wl.draft, bt, bd, B, H + N + g + 4, g)
    tau = torch.from_numpy(tau_np).cuda()
    mk = torch.from_numpy(mk_np).cuda()
    outs = s._outputs(B, N)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    fl = T.TPPSD_FLAG_HOST_LOOP if args.host_loop else 0

    def step_sd():
        T.tppsd_prefill(s.ctx, B, tau, mk, H, stream)
        T.tppsd_sample(s.ctx, B, N, g, 1234, fl, *outs, stream)

    def step_ar():
        T.tppsd_prefill(s.ctx, B, tau, mk, H, stream)
        T.tppsd_sample_autoregressive(s.ctx, B, N, 1234, fl, *outs, stream)

    def timed(step, K, W):
        for _ in range(W):
            step()
        barrier()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(K)]
        for e0, e1 in ev:
            flush.fill_(1.0)                 # evict L2 between timed steps (not timed)
            e0.record(stream)
            step()
            e1.record(stream)
        barrier()
        ms = sum(e0.elapsed_time(e1) for e0, e1 in ev) / K
        return max_over_ranks(ms, world, "cuda")

    with ClockSampler(local) as clk:
        ms_sd = timed(step_sd, args.steps, args.warmup)
    _, st_sd = T.tppsd_get_stats(s.ctx)
    # the AR comparator: same warm-up, up to 10 timed steps (~70 ms each)
    ms_ar = timed(step_ar, max(1, min(args.steps, 10)), args.warmup)
    _, st_ar = T.tppsd_get_stats(s.ctx)

    # Poisson draft (App. D.3) in place of the draft model, fitted by maximum
    # likelihood on a pilot AR sample of the target (64 events per sequence)
    pilot = s._outputs(B, 64)
    T.tppsd_prefill(s.ctx, B, tau, mk, H, stream)
    T.tppsd_sample_autoregressive(s.ctx, B, 64, 99, 0, *pilot, stream)
    rate, probs = fit_poisson_draft(pilot[0].cpu().numpy(), pilot[2].cpu().numpy(), wl.target.n_marks)

    def step_pois():
        T.tppsd_prefill(s.ctx, B, tau, mk, H, stream)
        T.tppsd_sample_poisson(s.ctx, B, N, g, rate, probs, 1234, fl, *outs, stream)

    ms_pois = timed(step_pois, max(1, min(args.steps, 3)), 1)
    _, st_pois = T.tppsd_get_stats(s.ctx)

    # end to end through the C ABI with pinned host buffers
    h_tau = torch.from_numpy(tau_np).pin_memory()
    h_mk = torch.from_numpy(mk_np).pin_memory()
    h_out = (torch.empty((B, N), dtype=torch.float32).pin_memory(),
             torch.empty((B, N), dtype=torch.float64).pin_memory(),
             torch.empty((B, N), dtype=torch.int32).pin_memory())

    def step_e2e():
        T.tppsd_prefill(s.ctx, B, h_tau, h_mk, H, stream)
        T.tppsd_sample(s.ctx, B, N, g, 1234, fl, *h_out, stream)

    ms_e2e = timed(step_e2e, max(1, min(args.steps, 3)), 1)
    h2d = B * H * (4 + 4)
    d2h = B * N * (4 + 8 + 4)

    # profiled call: CUDA events around every kernel launch
    T.tppsd_prefill(s.ctx, B, tau, mk, H, stream)
    T.tppsd_sample(s.ctx, B, N, g, 1234, T.TPPSD_FLAG_PROFILE, *outs, stream)
    kt = T.tppsd_kernel_times(s.ctx)
    _, st_prof = T.tppsd_get_stats(s.ctx)
    peaks = load_peaks()
    roof, per_class = roofline(kt, st_prof, wl, peaks)

    events = world * B * N
    value = job_rate(world, B, N, ms_sd)
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_sd, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic", "config": {**workload_config(wl, wl.seed),
                                        "launch": "host loop" if args.host_loop else "one CUDA graph per call"},
        "mean_accepted_per_verify": round(st_sd["accepted"] / max(st_sd["rounds"], 1), 3),
        "alpha": round(st_sd["accepted"] / max(st_sd["drafted"], 1), 4),
        "rounds": st_sd["loop_iters"],
        "ar": {"value": round(events / (ms_ar / 1e3), 1), "unit": UNIT, "ms_per_step": round(ms_ar, 3),
               "rounds": st_ar["loop_iters"]},
        "speedup_vs_ar": round(ms_ar / ms_sd, 3),
        "poisson_draft": {"value": round(events / (ms_pois / 1e3), 1), "unit": UNIT,
                          "ms_per_step": round(ms_pois, 3), "gamma": g, "rate": round(rate, 5),
                          "mean_accepted_per_verify": round(st_pois["accepted"] / max(st_pois["rounds"], 1), 3),
                          "alpha": round(st_pois["accepted"] / max(st_pois["drafted"], 1), 4),
                          "speedup_vs_ar": round(ms_ar / ms_pois, 3),
                          "fit": "MLE on a pilot AR sample of the target, 64 events per sequence"},
        "e2e": {"value": round(events / (ms_e2e / 1e3), 1), "unit": UNIT, "ms_per_step": round(ms_e2e, 3),
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": args.steps * (st_sd["kernel_launches"] + st_sd["prefill_launches"]),
        "clocks": clk.summary(),
        "roofline": roof,
        "path_roofline": path_roofline(per_class, ms_sd),
        "kernel_roofline": {k: {kk: v[kk] for kk in ("bound", "achieved", "peak", "unit", "frac",
                                                     "per_launch_ms", "share_of_device_time")}
                            for k, v in sorted(per_class.items(), key=lambda kv: -kv[1]["share_of_device_time"])},
        "kernel_ms": {k: round(v[0], 3) for k, v in kt.items() if v[1]},
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_oracle_rate(wl, bt, bd, tau_np, mk_np)
    s.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
