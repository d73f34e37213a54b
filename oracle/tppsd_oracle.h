/*
 * ORACLE -- test infrastructure only.
 *
 * A plain, slow, fp64 CPU restatement of TPP-SD (arxiv 2507.09252):
 * the CDF-based Transformer TPP of Sec. 4.2, naive autoregressive sampling
 * (Sec. 4.2, App. A.1), and the draft/verify/resample sampler of Sec. 4.3,
 * Alg. 1, Eq. 3-4 and Theorem 1.  Only tests/, __graft_entry__.smoke() and
 * bench.py's cpu_baseline / reference leg may load it.  It shares no code,
 * header, table or helper with the CUDA library.
 *
 * Each function cites the passage of the paper it follows; where the paper
 * is silent the reading taken is stated beside the code.
 */
#ifndef TPPSD_ORACLE_H
#define TPPSD_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* cfg[8] = {layers, d_model, heads, d_ffn, n_mix, n_marks, dtype, encoder};
 * dtype 0 = fp64 everywhere, 1 = bf16 rounding emulated at the GEMM inputs
 * and of Q/K/V (the points the CUDA path rounds at), all else fp64;
 * encoder 0 = THP, 1 = SAHP, 2 = AttNHP (App. D.4). */

/* Philox4x32-10 (Salmon et al., SC'11): one block of four 32-bit words. */
void oracle_philox4x32(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
/* The four uniforms in (0,1) of slot (seed, seq, pos, block). */
void oracle_uniforms(uint64_t seed, uint32_t seq, uint32_t pos, uint32_t block, double u[4]);

/* The model's temporal encoding z(t) (THP, SAHP or AttNHP form), d values. */
int oracle_model_temporal_encoding(const int32_t cfg[8], const float *blob, int64_t blob_floats,
                                   double t, double *out);

/* Teacher-forced heads: for every sequence b and position i in 0..len-2 the
 * head computed after encoding events 0..i (it predicts event i+1).  Head
 * row layout: [log w (M) | mu (M) | s = log sigma (M) | log f (K)].
 * out_heads has B*len*(3M+K) doubles; row i = len-1 is left untouched.
 * out_logg / out_logf (B*len, may be NULL) get log g(tau_i | h_{i-1}) and
 * log f(k_i | h_{i-1}) for i >= 1 and NaN at i = 0. */
int oracle_score(const int32_t cfg[8], const float *blob, int64_t blob_floats,
                 int32_t B, int32_t len, const float *tau, const int32_t *marks,
                 double *out_heads, double *out_logg, double *out_logf,
                 int32_t recompute, int32_t nthreads);

/* Naive autoregressive sampling from the target (Sec. 4.2).  History
 * tau/marks are [B][H]; outputs [B][N]: inter-event time, absolute time,
 * mark, and the smallest decision margin taken at that event.  seq_ids
 * (may be NULL = 0..B-1) gives each row's sequence index, which keys its
 * random slots. */
int oracle_sample_ar(const int32_t cfgT[8], const float *blobT, int64_t nT,
                     int32_t B, int32_t H, const float *hist_tau, const int32_t *hist_marks,
                     int32_t N, uint64_t seed, int32_t recompute, const int32_t *seq_ids,
                     double *out_tau, double *out_t, int32_t *out_k, double *out_margin,
                     int32_t nthreads);

/* TPP-SD (Sec. 4.3, Alg. 1).  flags bit 0 = no bonus event after a fully
 * accepted draft.  stats[B][5] = rounds, drafted, accepted, resample
 * iterations, resample-cap hits. */
int oracle_sample_sd(const int32_t cfgT[8], const float *blobT, int64_t nT,
                     const int32_t cfgD[8], const float *blobD, int64_t nD,
                     int32_t B, int32_t H, const float *hist_tau, const int32_t *hist_marks,
                     int32_t N, int32_t gamma, uint64_t seed, uint32_t flags, int32_t recompute,
                     const int32_t *seq_ids,
                     double *out_tau, double *out_t, int32_t *out_k, double *out_margin,
                     int64_t *stats, int32_t nthreads);

/* End-time forms (Alg. 1's stop rule): a sequence ends once its last event
 * lies beyond t_end or after N generated events; out_count[b] (may be NULL)
 * gets the number of generated events with t <= t_end, which fill the first
 * out_count[b] slots of the [B][N] outputs (later slots: NaN / -1).  The
 * forms above are these with t_end = +inf. */
int oracle_sample_ar_until(const int32_t cfgT[8], const float *blobT, int64_t nT,
                           int32_t B, int32_t H, const float *hist_tau, const int32_t *hist_marks,
                           int32_t N, double t_end, uint64_t seed, int32_t recompute,
                           const int32_t *seq_ids, double *out_tau, double *out_t, int32_t *out_k,
                           double *out_margin, int32_t *out_count, int32_t nthreads);
int oracle_sample_sd_until(const int32_t cfgT[8], const float *blobT, int64_t nT,
                           const int32_t cfgD[8], const float *blobD, int64_t nD,
                           int32_t B, int32_t H, const float *hist_tau, const int32_t *hist_marks,
                           int32_t N, double t_end, int32_t gamma, uint64_t seed, uint32_t flags,
                           int32_t recompute, const int32_t *seq_ids,
                           double *out_tau, double *out_t, int32_t *out_k, double *out_margin,
                           int32_t *out_count, int64_t *stats, int32_t nthreads);
/* TPP-SD with the Poisson draft of App. D.3: a homogeneous Poisson process
 * of rate lambda > 0 proposes the inter-event times (density
 * lambda exp(-lambda tau)) and marks are drafted iid from p_marks[K]
 * (normalised here; entries >= 0); the target's verification, resampling
 * (Theorem 1 against the exponential density, Eq. 4 against p) and bonus
 * are those of oracle_sample_sd.  Draft slot: block 0 at the event's
 * position, tau = -log(u_comp) / lambda, mark from p with u_mark.  Outputs
 * and stop rule as oracle_sample_sd_until.  Returns -1 on a bad lambda or
 * p. */
int oracle_sample_sd_poisson_until(const int32_t cfgT[8], const float *blobT, int64_t nT,
                                   int32_t B, int32_t H, const float *hist_tau,
                                   const int32_t *hist_marks, int32_t N, double t_end,
                                   int32_t gamma, double lambda, const double *p_marks,
                                   uint64_t seed, uint32_t flags, int32_t recompute,
                                   const int32_t *seq_ids, double *out_tau, double *out_t,
                                   int32_t *out_k, double *out_margin, int32_t *out_count,
                                   int64_t *stats, int32_t nthreads);
/* The Poisson draft's own draws (slot block 0 of positions 0..n-1 of
 * sequence 0), and Theorem 1 against it for a fixed target head (M
 * components, no marks). */
int oracle_sample_poisson(double lambda, int32_t K, const double *p, int32_t n, uint64_t seed,
                          double *out_tau, int32_t *out_k);
int oracle_resample_time_poisson(int32_t M, const double *headT, double lambda, int32_t n,
                                 uint64_t seed, double *out_tau, int32_t *iters);
/* Toy target (head = tableT[previous mark]) with the Poisson draft. */
int oracle_toy_sd_poisson(int32_t M, int32_t K, const double *tableT, double lambda,
                          const double *p_marks, int32_t B, int32_t N, int32_t gamma, uint64_t seed,
                          uint32_t flags, double *out_tau, int32_t *out_k, int64_t *stats);

/* Survival term log S(t_end - t_{len-1}) of each sequence's len events, from
 * the head after the last event (Sec. 3.1, Eq. 2). */
int oracle_score_survival(const int32_t cfg[8], const float *blob, int64_t blob_floats,
                          int32_t B, int32_t len, const float *tau, const int32_t *marks,
                          double t_end, double *out_logS, int32_t recompute, int32_t nthreads);
/* log(1 - G(u)) for the log-normal mixture of one head; 0 for u <= 0. */
double oracle_log_survival(int32_t M, const double *hd, double u);

/* Pieces on fixed heads (same row layout as oracle_score; M, K given). */
double oracle_log_g(int32_t M, const double *head, double tau);
double oracle_log_f(int32_t M, const double *head, int32_t k);
/* n direct draws (Sec. 4.2 / App. A.1); draw i uses slot (seed, 0, i, 0). */
void oracle_sample_head(int32_t M, int32_t K, const double *head, int32_t n, uint64_t seed,
                        double *out_tau, int32_t *out_k);
/* n draws from g' = norm(max(0, g_T - g_D)) by Theorem 1; draw i uses slots
 * (seed, 0, i, 2 + iteration).  iters (may be NULL) receives the count. */
void oracle_resample_time(int32_t M, const double *headT, const double *headD, int32_t n,
                          uint64_t seed, double *out_tau, int32_t *iters);
/* n draws from f' = norm(max(0, f_T - f_D)) (Eq. 4); draw i uses u_markres of
 * slot (seed, 0, i, 1). */
void oracle_resample_mark(int32_t M, int32_t K, const double *headT, const double *headD,
                          int32_t n, uint64_t seed, int32_t *out_k);

/* TPP-SD and AR on a toy model whose next-event head is a table indexed by
 * the previous event's mark: tables [K][3M+K].  One initial event (t=0 is not
 * an event: tau_0 = 1, mark 0).  Same slot layout as the transformer path. */
int oracle_toy_sd(int32_t M, int32_t K, const double *tableT, const double *tableD,
                  int32_t B, int32_t N, int32_t gamma, uint64_t seed, uint32_t flags,
                  double *out_tau, int32_t *out_k, int64_t *stats);
int oracle_toy_ar(int32_t M, int32_t K, const double *tableT, int32_t B, int32_t N,
                  uint64_t seed, double *out_tau, int32_t *out_k);

/* Temporal encoding z(t) (App. D.4, THP form) for tests: out[d]. */
void oracle_temporal_encoding(int32_t d, double t, double *out);
/* Round to bf16 (nearest, ties to even), for tests. */
double oracle_round_bf16(double x);

#ifdef __cplusplus
}
#endif
#endif
