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

    def sample_until(self, t_end, max_events, gamma, seed, flags=0, batch=None, stream=None):
        """TPP-SD until the end time t_end (Alg. 1's stop rule) or max_events;
        count[b] kept events (t <= t_end) fill the first slots."""
        torch = self.torch
        B = self.batch if batch is None else batch
        tau, t, k = self._outputs(B, max_events)
        cnt = torch.empty(B, dtype=torch.int32, device="cuda")
        T.tppsd_sample_until(self.ctx, B, t_end, max_events, gamma, seed, flags, tau, t, k, cnt, stream)
        return dict(tau=tau, t=t, k=k, count=cnt)

    def sample_ar_until(self, t_end, max_events, seed, flags=0, batch=None, stream=None):
        torch = self.torch
        B = self.batch if batch is None else batch
        tau, t, k = self._outputs(B, max_events)
        cnt = torch.empty(B, dtype=torch.int32, device="cuda")
        T.tppsd_sample_autoregressive_until(self.ctx, B, t_end, max_events, seed, flags, tau, t, k,
                                            cnt, stream)
        return dict(tau=tau, t=t, k=k, count=cnt)

    def sample_poisson(self, n_events, gamma, rate, mark_probs, seed, flags=0, batch=None,
                       stream=None):
        """TPP-SD with the Poisson draft of App. D.3 (rate, mark_probs)."""
        B = self.batch if batch is None else batch
        tau, t, k = self._outputs(B, n_events)
        T.tppsd_sample_poisson(self.ctx, B, n_events, gamma, rate, mark_probs, seed, flags, tau, t, k,
                               stream)
        return dict(tau=tau, t=t, k=k)

    def sample_poisson_until(self, t_end, max_events, gamma, rate, mark_probs, seed, flags=0,
                             batch=None, stream=None):
        torch = self.torch
        B = self.batch if batch is None else batch
        tau, t, k = self._outputs(B, max_events)
        cnt = torch.empty(B, dtype=torch.int32, device="cuda")
        T.tppsd_sample_poisson_until(self.ctx, B, t_end, max_events, gamma, rate, mark_probs, seed,
                                     flags, tau, t, k, cnt, stream)
        return dict(tau=tau, t=t, k=k, count=cnt)

    def score_until(self, which, tau, marks, t_end, heads=True, stream=None):
        """Eq. 2 on the window [0, t_end]: per-event terms as score() plus the
        survival term log S(t_end - t_last) per sequence (fp64)."""
        torch = self.torch
        tau = self._dev(tau, torch.float32)
        mk = self._dev(marks, torch.int32)
        B, n = tau.shape
        cfg = self.target if which == 0 else self.draft
        W = 3 * cfg.n_mix + cfg.n_marks
        hd = torch.full((B, n, W), float("nan"), device="cuda") if heads else None
        lg = torch.empty((B, n), device="cuda")
        lf = torch.empty((B, n), device="cuda")
        ls = torch.empty(B, dtype=torch.float64, device="cuda")
        T.tppsd_score_until(self.ctx, which, B, n, tau, mk, t_end, hd, lg, lf, ls, stream)
        self.batch = 0
        return hd, lg, lf, ls

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

    def trace(self, batch, n_events):
        """[batch][n_events][4] verify decisions of the last call made with
        TPPSD_FLAG_DEBUG_TRACE: time-test margin, mark-test margin, decision
        code (1 accepted, 2 time redrawn, 4 mark redrawn, 8 bonus), round."""
        return T.tppsd_get_trace(self.ctx, batch, n_events)


def fit_poisson_draft(hist_tau, hist_marks, n_marks, t_window=None):
    """Maximum-likelihood Poisson draft of App. D.3 from observed sequences
    (tppsd_fit_poisson_draft): rate = events / total observation window
    (each sequence's window t_window[b], default the time of its last event),
    mark probabilities = mark frequencies.  Fitting the draft is set-up, like
    loading weights; it is not part of sampling."""
    return T.tppsd_fit_poisson_draft(hist_tau, hist_marks, n_marks, t_window)
