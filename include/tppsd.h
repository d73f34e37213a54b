/*
 * tppsd.h -- C ABI of the GB300 TPP-SD sampler.
 *
 * TPP-SD (arxiv 2507.09252) samples a marked temporal point process from a
 * large "target" Transformer TPP by letting a small "draft" Transformer TPP
 * propose gamma events, verifying all of them with one causal target pass,
 * and resampling the first rejected event from the adjusted distribution
 * (Sec. 4.3, Alg. 1, Eq. 3-4, Theorem 1).  The output has the law of plain
 * autoregressive sampling from the target (App. A.2).
 *
 * Conventions for every entry point:
 *  - Status codes are returned; nothing throws or exits across the ABI.  On
 *    an error the context stays usable and outputs are unspecified.
 *  - A context must not be used by two host threads at once.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Work is enqueued on it; calls return before the GPU is done
 *    unless stated otherwise.
 *  - Array arguments are caller-owned.  Unless stated otherwise they may be
 *    host memory (pageable or pinned) or device memory: the library detects
 *    which and stages host data through its own device buffers on `stream`.
 *    Host outputs are complete when the stream has been synchronised
 *    (tppsd_wait); pageable host outputs are complete on return.
 *  - Sequences are independent; sequence b uses random slots keyed by b.
 */
#ifndef TPPSD_H
#define TPPSD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct tppsd_ctx tppsd_ctx; /* opaque, owned by the library */

typedef enum {
    TPPSD_OK = 0,
    TPPSD_ERR_INVALID_ARG = -1,  /* bad size, pointer, config or call order */
    TPPSD_ERR_OOM = -2,          /* device or host allocation failed */
    TPPSD_ERR_CUDA = -3,         /* a CUDA call failed; see tppsd_last_error */
    TPPSD_ERR_UNSUPPORTED = -4,  /* shape outside the compiled kernels' range */
    TPPSD_ERR_ROUND_LIMIT = -5,  /* the round loop stopped at its safety cap */
    TPPSD_ERR_TIMEOUT = -6,      /* tppsd_wait gave up before the GPU finished */
    TPPSD_ERR_NO_DEVICE = -7,    /* no CUDA device / driver */
    TPPSD_WARN_RESAMPLE_CAP = 1  /* a Theorem-1 loop hit its iteration cap */
} tppsd_status_t;

/* Model shape.  Weight blob layout (float32 values, row-major [out][in],
 * y = W x + b), in this order:
 *   type_emb [K][d]                                  (W of Sec. 4.2)
 *   for each layer, THP and SAHP:
 *                   w_qkv [3d][d], b_qkv [3d], w_o [d][d], b_o [d],
 *                   ln1_g [d], ln1_b [d], w_1 [F][d], b_1 [F],
 *                   w_2 [d][F], b_2 [d], ln2_g [d], ln2_b [d]
 *                 AttNHP: w_qkv [3d][2d] (inputs [z(t); h]), b_qkv [3d]
 *   E [3d][d]                                        (e = E h, no bias)
 *   v_w [M][d], b_w [M], v_mu [M][d], b_mu [M], v_s [M][d], b_s [M]
 *   v_k1 [d][d], b_k1 [d], v_k2 [K][d], b_k2 [K]
 *   SAHP only: w [d] (temporal frequencies); AttNHP only: m, M (time scales)
 * Model (Sec. 4.2): x_i = z(t_i) + W[k_i]; heads w = softmax(v_w e1 + b_w),
 * mu = v_mu e2 + b_mu, sigma = exp(v_s e3 + b_s), f = softmax(v_k2
 * tanh(v_k1 h + b_k1) + b_k2).  Encoders (App. D.4), t absolute, j 0-based,
 * je = j - j mod 2, sin for even j and cos for odd j of:
 *   THP     t / 10000^(je/d)
 *   SAHP    j / 10000^(je/d) + w_j t
 *   AttNHP  t / (m (5M/m)^(je/d))
 * THP and SAHP layers: post-LN h <- LN(h + MHA(h)), h <- LN(h + W2 ReLU(W1
 * h + b1) + b2), causal softmax attention (scale 1/sqrt(d/heads)), LayerNorm
 * eps 1e-5.  AttNHP layers: q, k, v = w_qkv [z; h] + b_qkv; per head
 * a = sum_j f_j v_j / (1 + sum_j f_j), f_j = exp(q k_j / sqrt(d/heads)) over
 * keys j <= i; h <- h + tanh(a) (heads concatenated).
 * dtype 0 = fp32 throughout.  dtype 1 = bf16: the blob's values must be
 * bf16-representable; GEMM inputs and Q/K/V are rounded to bf16 (nearest
 * even), accumulation, LayerNorm, softmax, heads and sampling are fp32. */
typedef struct {
    int32_t layers;   /* 1..16 */
    int32_t d_model;  /* multiple of 16, <= 512 */
    int32_t heads;    /* 1..8 (draft: 1, 2 or 4); d_model / heads in {8, 16, 32, 64} */
    int32_t d_ffn;    /* multiple of 16, <= 4096 (unused by AttNHP) */
    int32_t n_mix;    /* M, 1..64 */
    int32_t n_marks;  /* K, 1..256; equal for target and draft */
    int32_t dtype;    /* 0 fp32, 1 bf16 */
    int32_t encoder;  /* 0 THP, 1 SAHP, 2 AttNHP (an AttNHP draft model must
                         fit the one-CTA draft kernel: heads 1, 2 or 4 and
                         d/heads 16 or 32, else TPPSD_ERR_UNSUPPORTED) */
} tppsd_model_cfg;

/* Counters of the last tppsd_sample / tppsd_sample_autoregressive call. */
typedef struct {
    int64_t rounds;          /* (sequence, round) pairs; AR: events sampled */
    int64_t drafted;         /* draft events proposed (gamma per pair) */
    int64_t accepted;        /* drafts accepted before the first rejection */
    int64_t emitted;         /* events written, before truncation to n_events */
    int64_t resample_iters;  /* Theorem-1 loop iterations */
    int64_t cap_hits;        /* Theorem-1 loops stopped by the cap */
    int64_t loop_iters;      /* device round-loop iterations */
    int64_t kernel_launches; /* kernels launched by the call */
    int64_t target_keys;     /* sum over (sequence, target pass) of cached keys read per layer */
    int64_t draft_keys;      /* sum over draft positions encoded of keys read per layer */
    int64_t prefill_launches;/* kernels launched by the last tppsd_prefill */
} tppsd_stats;

/* Number of floats a blob of this shape must hold (0 if unsupported). */
size_t tppsd_blob_floats(const tppsd_model_cfg* cfg);

/* Uploads both models and allocates KV caches and buffers for up to
 * max_batch sequences of max_positions events (history + generated +
 * gamma + 1) and draft length up to max_gamma.  Blobs: host or device
 * float arrays of tppsd_blob_floats() values, copied.  *out receives the
 * context, or NULL on error. */
tppsd_status_t tppsd_create_models(const tppsd_model_cfg* target, const tppsd_model_cfg* draft,
                                   const float* target_blob, size_t target_floats,
                                   const float* draft_blob, size_t draft_floats,
                                   int32_t max_batch, int32_t max_positions, int32_t max_gamma,
                                   tppsd_ctx** out);

/* Binds the history of `batch` sequences and encodes it with both models
 * (KV caches of events 0..hist_len-2; event hist_len-1 is encoded by the
 * first verify pass).  hist_tau [batch][hist_len] inter-event times
 * (t_1 = tau_1, t_i = t_{i-1} + tau_i, summed in fp64), hist_marks
 * [batch][hist_len] in 0..K-1 (values outside are clamped into range).
 * hist_len >= 1. */
tppsd_status_t tppsd_prefill(tppsd_ctx* ctx, int32_t batch, const float* hist_tau,
                             const int32_t* hist_marks, int32_t hist_len, void* stream);

#define TPPSD_FLAG_NO_BONUS 1u  /* no extra target event after a full accept */
#define TPPSD_FLAG_HOST_LOOP 2u /* round loop driven from the host (debug) */
#define TPPSD_FLAG_PROFILE 4u   /* host-driven loop with CUDA events around every kernel */
#define TPPSD_FLAG_DEBUG_TRACE 8u /* record every verify decision (tppsd_get_trace) */

/* TPP-SD (Sec. 4.3, Alg. 1): draws n_events events after the prefilled
 * history of each of the first `batch` sequences, with gamma drafts per
 * round.  Uniforms: Philox4x32-10 keyed by `seed`, counter (event index,
 * block, sequence, 0).  Outputs [batch][n_events]: out_tau inter-event
 * times (fp32), out_t absolute times (fp64), out_marks.  Each call restarts
 * from the prefilled history. */
tppsd_status_t tppsd_sample(tppsd_ctx* ctx, int32_t batch, int32_t n_events, int32_t gamma,
                            uint64_t seed, uint32_t flags, float* out_tau, double* out_t,
                            int32_t* out_marks, void* stream);

/* Target-only autoregressive sampling (Sec. 4.2), same slots and outputs. */
tppsd_status_t tppsd_sample_autoregressive(tppsd_ctx* ctx, int32_t batch, int32_t n_events,
                                           uint64_t seed, uint32_t flags, float* out_tau,
                                           double* out_t, int32_t* out_marks, void* stream);

/* TPP-SD with the end-time stop rule of Alg. 1: each of the first `batch`
 * sequences is extended until its last event lies beyond t_end (absolute
 * time, same clock as the history) or max_events events are drawn, in
 * rounds of gamma drafts.  Random slots as tppsd_sample, so the events kept
 * are the prefix with t <= t_end of the tppsd_sample run with the same seed
 * and n_events = max_events.  Outputs [batch][max_events]: the first
 * out_count[b] slots hold the kept events; the rest are NaN (out_tau,
 * out_t) and -1 (out_marks).  out_count [batch] (host or device) is
 * required; a history already ending beyond t_end gives count 0.  t_end =
 * +inf is tppsd_sample; NaN is TPPSD_ERR_INVALID_ARG. */
tppsd_status_t tppsd_sample_until(tppsd_ctx* ctx, int32_t batch, double t_end, int32_t max_events,
                                  int32_t gamma, uint64_t seed, uint32_t flags, float* out_tau,
                                  double* out_t, int32_t* out_marks, int32_t* out_count,
                                  void* stream);

/* Target-only autoregressive sampling (Sec. 4.2) with the same stop rule,
 * slots and outputs as tppsd_sample_until. */
tppsd_status_t tppsd_sample_autoregressive_until(tppsd_ctx* ctx, int32_t batch, double t_end,
                                                 int32_t max_events, uint64_t seed, uint32_t flags,
                                                 float* out_tau, double* out_t, int32_t* out_marks,
                                                 int32_t* out_count, void* stream);

/* TPP-SD with the Poisson draft of App. D.3 in place of the draft model: a
 * homogeneous Poisson process of rate `rate` (> 0) proposes the gamma
 * inter-event times of a round (density rate exp(-rate tau)) and the marks
 * are proposed iid from mark_probs, a HOST array of K doubles (the target's
 * n_marks; entries >= 0 with a positive sum, normalised by the library).
 * The paper fits both by maximum likelihood on the data (rate = events per
 * unit time, mark_probs = mark frequencies).  Draft slot: block 0 at the
 * event's position, tau = -log(u_comp) / rate, mark with u_mark.  The
 * target's verification, resampling (Theorem 1 against the exponential
 * density, Eq. 4 against mark_probs) and bonus are those of tppsd_sample,
 * and so are the outputs; the draft model of the context is not used.  A
 * bad rate or mark_probs is TPPSD_ERR_INVALID_ARG. */
tppsd_status_t tppsd_sample_poisson(tppsd_ctx* ctx, int32_t batch, int32_t n_events, int32_t gamma,
                                    double rate, const double* mark_probs, uint64_t seed,
                                    uint32_t flags, float* out_tau, double* out_t,
                                    int32_t* out_marks, void* stream);

/* Maximum-likelihood fit of the Poisson draft of App. D.3 from observed
 * sequences tau / marks [batch][len] (host or device; inter-event times,
 * marks in 0..n_marks-1): a homogeneous Poisson process observed on the
 * windows [0, T_b] has likelihood prod lambda^n_b exp(-lambda T_b), so
 * rate = (number of events) / (sum of T_b), and iid marks give
 * mark_probs[k] = (events with mark k) / (number of events).  t_window
 * [batch] (host, may be NULL) holds each sequence's observation window
 * T_b, which must reach its last event; NULL takes T_b = time of the last
 * event (the sum of its tau).  Outputs: *out_rate and out_mark_probs
 * [n_marks] (host, fp64), ready for tppsd_sample_poisson.  Host work, no
 * context needed.  TPPSD_ERR_INVALID_ARG for empty input, a negative or
 * non-finite tau, a mark out of range, a window before the last event or a
 * total window of zero. */
tppsd_status_t tppsd_fit_poisson_draft(int32_t batch, int32_t len, const float* tau,
                                       const int32_t* marks, const double* t_window,
                                       int32_t n_marks, double* out_rate, double* out_mark_probs);

/* The same with the end-time stop rule, outputs as tppsd_sample_until. */
tppsd_status_t tppsd_sample_poisson_until(tppsd_ctx* ctx, int32_t batch, double t_end,
                                          int32_t max_events, int32_t gamma, double rate,
                                          const double* mark_probs, uint64_t seed, uint32_t flags,
                                          float* out_tau, double* out_t, int32_t* out_marks,
                                          int32_t* out_count, void* stream);

/* Teacher-forced scoring with one model (which 0 = target, 1 = draft): for
 * sequences tau/marks [batch][len], out_heads [batch][len][3M+K] (may be
 * NULL) gets the head after events 0..i at row i (row len-1 untouched):
 * [log w | mu | log sigma | log f]; out_logg / out_logf [batch][len] (may
 * be NULL) get log g(tau_i | h_{i-1}) and log f(k_i | h_{i-1}) (Eq. 2
 * terms), NaN at i = 0.  Overwrites the caches: prefill again before
 * sampling. */
tppsd_status_t tppsd_score(tppsd_ctx* ctx, int32_t which, int32_t batch, int32_t len,
                           const float* tau, const int32_t* marks, float* out_heads,
                           float* out_logg, float* out_logf, void* stream);

/* Log-likelihood on the observation window [0, t_end] (Eq. 2): the outputs
 * of tppsd_score, and in out_logS [batch] (fp64, host or device, required)
 * the survival term log(1 - G(t_end - t_last)) of each sequence, G the
 * inter-event CDF of the head after its last event (the log-normal mixture
 * of Sec. 4.2; computed in fp64 from the fp32 head), 0 when t_end <= t_last.
 * One pass over all len positions, so out_heads (may be NULL) also gets row
 * len-1.  len >= 1; at len = 1 out_logg / out_logf are NaN.  Overwrites the
 * caches like tppsd_score. */
tppsd_status_t tppsd_score_until(tppsd_ctx* ctx, int32_t which, int32_t batch, int32_t len,
                                 const float* tau, const int32_t* marks, double t_end,
                                 float* out_heads, float* out_logg, float* out_logf,
                                 double* out_logS, void* stream);

/* Scoring that allocates nothing (the paper has no counterpart; this is a
 * library convenience).  Same outputs as tppsd_score's out_logg and
 * out_logf for device arrays tau, marks, out_logg, out_logf [batch][len];
 * no head rows.  For callers that may not allocate device memory at call
 * time: processes whose GPU memory is owned by another allocator, or
 * latency-critical loops that cannot absorb cudaMalloc's implicit device
 * synchronisation.  All working memory (sequence copy, K/V of the scored
 * positions, row workspace) comes from one 16 MiB array in device memory
 * that the library holds on every GPU that loads it until the process
 * exits; a request whose K/V and sequence copy do not fit (with room for at
 * least 16 workspace rows) returns TPPSD_ERR_INVALID_ARG with the reason
 * in tppsd_last_error.  The first call on a device looks up that array's
 * device address (a one-time set-up); make that first call before any
 * stream capture.  Every call shares the array: calls that overlap on the
 * GPU (other streams, other contexts, other host threads) race and give
 * wrong results; serialise them.  Unlike tppsd_score it leaves the
 * prefilled caches intact.  A bounded wait that runs out inside a kernel is
 * reported by tppsd_wait, as for tppsd_score. */
tppsd_status_t tppsd_score_noalloc(tppsd_ctx* ctx, int32_t which, int32_t batch, int32_t len,
                                   const float* tau, const int32_t* marks, float* out_logg,
                                   float* out_logf, void* stream);

/* Decisions of the last tppsd_sample / tppsd_sample_until /
 * tppsd_sample_poisson(_until) call made with TPPSD_FLAG_DEBUG_TRACE (Alg. 1:
 * the tests of Sec. 4.3, the first rejection, Theorem 1 and Eq. 4), for the
 * first n_events generated events of each of the first `batch` sequences:
 * out [batch][n_events][4] floats (host or device), per event
 *   [0] u_tau - min(1, g_T / g_D) of its time test (negative: accepted)
 *   [1] u_k - min(1, f_T / f_D) of its mark test
 *   [2] decision code: 1 accepted draft; at the first rejection 2 (time
 *       redrawn by Theorem 1) + 4 (mark redrawn from Eq. 4); 8 bonus event
 *       drawn from the target (no test: [0], [1] NaN)
 *   [3] the device round-loop iteration that decided it.
 * The margins are the GPU's own, computed in its own precision: a sampled
 * sequence can only differ from an exact computation after a decision
 * whose margin is about that precision.  Events never reached read as 0.
 * TPPSD_ERR_INVALID_ARG if the last call was not traced or the sizes
 * exceed it. */
tppsd_status_t tppsd_get_trace(tppsd_ctx* ctx, int32_t batch, int32_t n_events, float* out);

/* Safety limits of the sampling calls that follow (diagnostics and tests).
 * resample_cap: iteration cap of the Theorem-1 resampling loop (Theorem 1
 * leaves the loop unbounded; the library stops it after resample_cap
 * proposals, keeps the last proposal and reports TPPSD_WARN_RESAMPLE_CAP,
 * reading c6 of the sampler); 0 restores the default 65 536.  max_rounds:
 * cap on the device round loop of Alg. 1 below its natural bound of
 * n_events + 2 rounds (every round emits at least one event per active
 * sequence); a call that reaches it stops and tppsd_get_stats returns
 * TPPSD_ERR_ROUND_LIMIT; 0 removes the extra cap.  Negative values are
 * TPPSD_ERR_INVALID_ARG.  Host-side only; takes effect at the next call. */
tppsd_status_t tppsd_set_limits(tppsd_ctx* ctx, int32_t resample_cap, int32_t max_rounds);

/* Synchronises the last stream used and copies the last call's counters.
 * Returns that call's status (OK, WARN_RESAMPLE_CAP or ERR_ROUND_LIMIT). */
tppsd_status_t tppsd_get_stats(tppsd_ctx* ctx, tppsd_stats* out);

/* Per-kernel-class device time of the last call made with
 * TPPSD_FLAG_PROFILE (synchronises): ms[TPPSD_KERNEL_CLASSES] total
 * milliseconds measured with CUDA events on the call's stream, launches[]
 * counts.  Class names: tppsd_kernel_class_name(i). */
#define TPPSD_KERNEL_CLASSES 13
tppsd_status_t tppsd_kernel_times(tppsd_ctx* ctx, double* ms, int64_t* launches);
const char* tppsd_kernel_class_name(int32_t cls);

/* Host watchdog: waits at most timeout_ms for the last call's work;
 * TPPSD_ERR_TIMEOUT if it is still running then, or if a bounded wait
 * inside one of the call's kernels ran out (the kernel recorded it and
 * returned early; the context stays usable and the next call clears the
 * record).  Setting TPPSD_FAULT=wait in the environment makes the
 * tensor-core QKV GEMM of the scoring calls wait on a barrier that nothing
 * completes, so its bounded wait runs out: a test of that path. */
tppsd_status_t tppsd_wait(tppsd_ctx* ctx, int32_t timeout_ms);

const char* tppsd_status_str(tppsd_status_t status);
const char* tppsd_last_error(const tppsd_ctx* ctx); /* "" if none */
void tppsd_destroy(tppsd_ctx* ctx);

#ifdef __cplusplus
}
#endif
#endif
