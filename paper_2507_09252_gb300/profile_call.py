"""Per-kernel-class timing of one sampling call.

    python -m paper_2507_09252_gb300.profile_call [--workload c2] [--calls 2]
                                                  [--mode sd|ar] [--host-loop]

Builds the workload's models and histories (seeded, synthetic), prefills,
and runs `--calls` sampling calls.  By default each call runs with
TPPSD_FLAG_PROFILE (every launch bracketed by CUDA events) and the
per-class totals are printed; with --host-loop the calls run the rounds
from a host loop without events, which is the form a per-launch profiler
(ncu) can attribute, since kernels inside a CUDA graph's conditional loop
are not visible to it.
"""
import argparse
import json
import sys

from . import configs as CF
from . import inputs as IN
from . import tppsd as T
from .sampler import Sampler

WORKLOADS = {"c1": CF.C1, "c2": CF.C2}


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="c2", choices=sorted(WORKLOADS))
    ap.add_argument("--calls", type=int, default=2,
                    help="calls to run; the per-class times are those of the last one "
                         "(the first call also pays one-time kernel loading)")
    ap.add_argument("--mode", default="sd", choices=["sd", "ar"])
    ap.add_argument("--host-loop", action="store_true")
    a = ap.parse_args(argv)
    import torch
    wl = WORKLOADS[a.workload]
    B, H, N, g = wl.batch, wl.hist_len, wl.n_events, wl.gamma
    bt, bd = IN.model_blob(wl.target, wl.seed, 0), IN.model_blob(wl.draft, wl.seed, 1)
    tau_np, mk_np = IN.histories(wl, seed=wl.seed)
    s = Sampler(wl.target, wl.draft, bt, bd, B, H + N + g + 4, g)
    tau, mk = torch.from_numpy(tau_np).cuda(), torch.from_numpy(mk_np).cuda()
    outs = s._outputs(B, N)
    st = torch.cuda.current_stream()
    flags = T.TPPSD_FLAG_HOST_LOOP if a.host_loop else T.TPPSD_FLAG_PROFILE
    for _ in range(a.calls):
        T.tppsd_prefill(s.ctx, B, tau, mk, H, st)
        if a.mode == "sd":
            T.tppsd_sample(s.ctx, B, N, g, 1234, flags, *outs, st)
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
