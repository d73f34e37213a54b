"""Convenience wrapper over the C ABI for torch users (marshalling only).

    s = Sampler(target_cfg, draft_cfg, blob_t, blob_d, max_batch=256,
                max_positions=H + N + gamma + 2, max_gamma=8)
    s.prefill(hist_tau, hist_marks)              # [B][H] tensors or arrays
    out = s.sample(n_events=512, gamma=8, seed=0)  # dict of CUDA tensors
"""
import numpy as np

from . import tppsd as T


class Sampler:
    def __init__(self, target, draft, blob_t, blob_d, max_batch, max_positions, max_gamma):
        import torch
        self.torch = torch
        self.target, self.draft = target, draft
        self.ctx = T.tppsd_create_models(target, draft, np.ascontiguousarray(blob_t, np.float32),
                                         np.ascontiguousarray(blob_d, np.float32), max_batch,
                                         max_positions, max_gamma)
        self.batch = 0

    def close(self):
        if self.ctx:
            T.tppsd_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _dev(self, a, dtype):
        torch = self.torch
        if isinstance(a, np.ndarray):
            a = torch.from_numpy(np.ascontiguousarray(a))
        return a.to(device="cuda", dtype=dtype).contiguous()

    def prefill(self, hist_tau, hist_marks, stream=None):
        tau = self._dev(hist_tau, self.torch.float32)
        mk = self._dev(hist_marks, self.torch.int32)
        B, H = tau.shape
        T.tppsd_prefill(self.ctx, B, tau, mk, H, stream)
        self.batch, self.hist_len = B, H
        self._keep = (tau, mk)  # alive until the stream has consumed them

    def _outputs(self, B, N):
        torch = self.torch
        return (torch.empty((B, N), dtype=torch.float32, device="cuda"),
                torch.empty((B, N), dtype=torch.float64, device="cuda"),
                torch.empty((B, N), dtype=torch.int32, device="cuda"))

    def sample(self, n_events, gamma, seed, flags=0, batch=None, out=None, stream=None):
        B = self.batch if batch is None else batch
        tau, t, k = out if out is not None else self._outputs(B, n_events)
        T.tppsd_sample(self.ctx, B, n_events, gamma, seed, flags, tau, t, k, stream)
        return dict(tau=tau, t=t, k=k)

    def sample_ar(self, n_events, seed, flags=0, batch=None, out=None, stream=None):
        B = self.batch if batch is None else batch
        tau, t, k = out if out is not None else self._outputs(B, n_events)
        T.tppsd_sample_autoregressive(self.ctx, B, n_events, seed, flags, tau, t, k, stream)
        return dict(tau=tau, t=t, k=k)

    def score(self, which, tau, marks, heads=True, stream=None):
        torch = self.torch
        tau = self._dev(tau, torch.float32)
        mk = self._dev(marks, torch.int32)
        B, n = tau.shape
        cfg = self.target if which == 0 else self.draft
        W = 3 * cfg.n_mix + cfg.n_marks
        hd = torch.full((B, n, W), float("nan"), device="cuda") if heads else None
        lg = torch.empty((B, n), device="cuda")
        lf = torch.empty((B, n), device="cuda")
        T.tppsd_score(self.ctx, which, B, n, tau, mk, hd, lg, lf, stream)
        self.batch = 0  # scoring overwrote the prefilled caches
        return hd, lg, lf

    def stats(self):
        return T.tppsd_get_stats(self.ctx)
