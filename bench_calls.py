"""Per-kernel-class timing of sampling calls, and a throughput mode for every
workload shape.

    python bench_calls.py [--workload c2] [--calls 2] [--mode sd|ar] [--host-loop]
    python bench_calls.py --time --workload c3 [--gamma 4] [--batch 16] [--draft 0]
                          [--encoder attnhp] [--hist-len 4096] [--n-events 256]

Builds the workload's models and histories (seeded, synthetic) and prefills.

Default: runs `--calls` sampling calls with TPPSD_FLAG_PROFILE (every launch
bracketed by CUDA events) and prints the per-class totals of the last one
(the first call also pays one-time kernel loading).  With --host-loop the
calls run the rounds from a host loop without events, the form a per-launch
profiler (ncu) can attribute: kernels inside a CUDA graph's conditional loop
are not visible to it.

--time: TPP-SD and target-only AR events/s of the graph-launched calls
(CUDA events, inputs resident, 2 warm-up + 3 timed calls each, L2 flushed
before each timed call), mean accepted drafts per verify and acceptance
rate, as one JSON line, with the draft and target-attention kernels against
the HBM peak (from one profiled call).  --gamma / --batch / --draft override
the workload's gamma, batch and draft model (an index into the workload's
draft sweep); --hist-len / --n-events its history and generated lengths
(a long history puts every round's context past that many keys).
--poisson: the draft is the Poisson process of App. D.3, fitted by maximum
likelihood on a pilot AR sample of the target (64 events per sequence).
"""
import argparse
import json
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

from paper_2507_09252_gb300 import configs as CF  # noqa: E402
from paper_2507_09252_gb300 import inputs as IN  # noqa: E402
from paper_2507_09252_gb300 import tppsd as T  # noqa: E402
from paper_2507_09252_gb300.sampler import Sampler  # noqa: E402

WORKLOADS = {"c1": CF.C1, "c2": CF.C2, "c3": CF.C3, "c4": CF.C4, "c5": CF.C5}


def _time_calls(torch, fn, flush, reps=3, warm=2):
    st = torch.cuda.current_stream()
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    tot = 0.0
    for _ in range(reps):
        flush.fill_(1.0)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(st)
        fn()
        e1.record(st)
        torch.cuda.synchronize()
        tot += e0.elapsed_time(e1)
    return tot / reps


def _hbm_peak():
    """Measured HBM copy bandwidth of this machine (GB/s), else the fallback."""
    try:
        with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"])
    except (OSError, KeyError, ValueError):
        return 6800.0


def attention_roofline(ms, launches, stats, wl):
    """The target attention class of one profiled call against the HBM
    peak, by bench.py's per-class formula."""
    import bench
    r = bench.class_roofline("attention", ms, launches, stats, wl, {"hbm_gbs": _hbm_peak()}, False)
    return {"us_per_launch": round(1e3 * ms / launches, 2), "bytes_per_launch": int(r["algorithmic_per_launch"]),
            "mean_keys_per_sequence": round(stats["target_keys"] / max(stats["rounds"], 1), 1),
            "achieved_GBps": r["achieved"], "frac_of_hbm": r["frac"]}


def _shape(cfg, fields):
    return " ".join(f"{n}{getattr(cfg, f)}" for n, f in fields)


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="c2", choices=sorted(WORKLOADS))
    ap.add_argument("--calls", type=int, default=2,
                    help="calls to run; the per-class times are those of the last one "
                         "(the first call also pays one-time kernel loading)")
    ap.add_argument("--mode", default="sd", choices=["sd", "ar"])
    ap.add_argument("--host-loop", action="store_true")
    ap.add_argument("--time", action="store_true")
    ap.add_argument("--gamma", type=int, default=None)
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--draft", type=int, default=None)
    ap.add_argument("--poisson", action="store_true")
    ap.add_argument("--hist-len", type=int, default=None)
    ap.add_argument("--n-events", type=int, default=None)
    ap.add_argument("--encoder", default=None, choices=["thp", "sahp", "attnhp"],
                    help="history encoder of both models (App. D.4); default: the workload's")
    a = ap.parse_args(argv)
    import torch
    wl = WORKLOADS[a.workload]
    if a.gamma is not None:
        wl = wl.with_(gamma=a.gamma)
    if a.batch is not None:
        wl = wl.with_(batch=a.batch)
    if a.draft is not None:
        wl = wl.with_(draft=wl.drafts[a.draft])
    if a.hist_len is not None:
        wl = wl.with_(hist_len=a.hist_len)
    if a.n_events is not None:
        wl = wl.with_(n_events=a.n_events)
    if a.encoder is not None:
        enc = {"thp": CF.THP, "sahp": CF.SAHP, "attnhp": CF.ATTNHP}[a.encoder]
        wl = wl.with_(target=CF.ModelCfg(**{**wl.target.__dict__, "encoder": enc}),
                      draft=CF.ModelCfg(**{**wl.draft.__dict__, "encoder": enc}))
    B, H, N, g = wl.batch, wl.hist_len, wl.n_events, wl.gamma
    bt, bd = IN.model_blob(wl.target, wl.seed, 0), IN.model_blob(wl.draft, wl.seed, 1)
    tau_np, mk_np = IN.histories(wl, seed=wl.seed)
    s = Sampler(wl.target, wl.draft, bt, bd, B, H + N + g + 4, g)
    tau, mk = torch.from_numpy(tau_np).cuda(), torch.from_numpy(mk_np).cuda()
    outs = s._outputs(B, N)
    st = torch.cuda.current_stream()
    from paper_2507_09252_gb300.sampler import fit_poisson_draft
    rate, probs = 1.0, None
    if a.poisson:  # MLE on a pilot AR sample of the target (the data it models)
        T.tppsd_prefill(s.ctx, B, tau, mk, H, st)
        pilot = s._outputs(B, min(N, 64))
        T.tppsd_sample_autoregressive(s.ctx, B, min(N, 64), 99, 0, *pilot, st)
        rate, probs = fit_poisson_draft(pilot[0].cpu().numpy(), pilot[2].cpu().numpy(),
                                        wl.target.n_marks)

    def sample_call(flags):
        if a.poisson:
            T.tppsd_sample_poisson(s.ctx, B, N, g, rate, probs, 1234, flags, *outs, st)
        else:
            T.tppsd_sample(s.ctx, B, N, g, 1234, flags, *outs, st)
    if a.time:
        flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device="cuda")

        def sd():
            T.tppsd_prefill(s.ctx, B, tau, mk, H, st)
            sample_call(0)

        def ar():
            T.tppsd_prefill(s.ctx, B, tau, mk, H, st)
            T.tppsd_sample_autoregressive(s.ctx, B, N, 1234, 0, *outs, st)

        ms_sd = _time_calls(torch, sd, flush)
        _, st_sd = T.tppsd_get_stats(s.ctx)
        ms_ar = _time_calls(torch, ar, flush, reps=2, warm=1)
        # the draft kernel against HBM: one profiled call gives its time per
        # round; its bytes are the draft K/V it reads per round (every key of
        # the context once per encoded position when the cache is streamed;
        # once per round when it stays in shared memory), counted by the
        # kernel (draft_keys, per layer)
        # The target's attention against HBM, from the same profiled call,
        # by bench.py's formula: K and V of every cached key once per
        # (sequence, layer), counted by the kernels (target_keys), plus the
        # Q rows read and the output rows written (CUDA-event time per
        # launch, launch gap included)
        draft = attn = None
        if not a.poisson:
            T.tppsd_prefill(s.ctx, B, tau, mk, H, st)
            sample_call(T.TPPSD_FLAG_PROFILE)
            torch.cuda.synchronize()
            _, st_p = T.tppsd_get_stats(s.ctx)
            kt = T.tppsd_kernel_times(s.ctx)
            ams, an = kt.get("attention", (0.0, 0))
            if an:
                attn = attention_roofline(ams, an, st_p, wl)
            kms, kn = kt.get("draft", (0.0, 0))
            if kn:
                eb = 2 if wl.draft.dtype == CF.BF16 else 4
                dcfg = wl.draft
                kv = st_p["draft_keys"] * dcfg.layers * 2 * dcfg.d_model * eb
                gbs = kv / (kms / 1e3) / 1e9
                peak = _hbm_peak()
                draft = {"us_per_round": round(1e3 * kms / kn, 2),
                         "kv_bytes_per_round": int(kv / kn),
                         "achieved_GBps": round(gbs, 1), "frac_of_hbm": round(gbs / peak, 4),
                         "peak_GBps": peak}
        layer = (("L", "layers"), ("d", "d_model"), ("h", "heads"), ("F", "d_ffn"))
        print(json.dumps({
            "workload": wl.name, "batch": B, "gamma": g, "n_events": N, "hist_len": H,
            "target": _shape(wl.target, layer + (("M", "n_mix"), ("K", "n_marks"))),
            "draft": f"Poisson rate {rate:.4g}" if a.poisson else _shape(wl.draft, layer),
            "encoder": ["THP", "SAHP", "AttNHP"][wl.target.encoder],
            "sd_events_per_s": round(B * N / (ms_sd / 1e3), 1), "sd_ms_per_call": round(ms_sd, 3),
            "ar_events_per_s": round(B * N / (ms_ar / 1e3), 1), "ar_ms_per_call": round(ms_ar, 3),
            "speedup_vs_ar": round(ms_ar / ms_sd, 3),
            "mean_accepted_per_verify": round(st_sd["accepted"] / max(st_sd["rounds"], 1), 3),
            "alpha": round(st_sd["accepted"] / max(st_sd["drafted"], 1), 4),
            "rounds": st_sd["loop_iters"], "draft_kernel": draft, "attention_kernel": attn,
            "note": "prefill included in both timed calls"}), flush=True)
        s.close()
        return 0
    flags = T.TPPSD_FLAG_HOST_LOOP if a.host_loop else T.TPPSD_FLAG_PROFILE
    for _ in range(a.calls):
        T.tppsd_prefill(s.ctx, B, tau, mk, H, st)
        if a.mode == "sd":
            sample_call(flags)
        else:
            T.tppsd_sample_autoregressive(s.ctx, B, N, 1234, flags, *outs, st)
    torch.cuda.synchronize()
    _, stats = T.tppsd_get_stats(s.ctx)
    if not a.host_loop:
        kt = T.tppsd_kernel_times(s.ctx)
        tot = sum(v[0] for v in kt.values()) or 1.0
        for k, (ms, n) in sorted(kt.items(), key=lambda kv: -kv[1][0]):
            if n:
                print(f"{k:12s} {ms:9.3f} ms {n:7d} launches {1e3 * ms / n:9.2f} us/launch "
                      f"{ms / tot:6.3f} of device time")
    print(json.dumps(stats))
    s.close()
    return 0


if __name__ == "__main__":
    sys.exit(main())
