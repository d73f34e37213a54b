/*
 * ORACLE -- test infrastructure only (see tppsd_oracle.h).
 *
 * Plain fp64 C.  Every function follows the paper passage it cites, in the
 * paper's order; nothing is blocked, fused or reordered.  Readings of points
 * the paper leaves open are marked "Reading:".
 *
 * Build: gcc -O2 -ffp-contract=off -fopenmp -fPIC -shared (oracle/build.py).
 * -ffp-contract=off keeps x86 and Arm results bit-identical.
 */
#include "tppsd_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define MAXM 64
#define MAXK 256
#define RESAMPLE_CAP 65536
#define FLAG_NO_BONUS 1u
#define LN_EPS 1e-5

static const double LOG_2PI = 1.8378770664093454835606594728112;
static const double TWO_PI = 6.283185307179586476925286766559;

/* ------------------------------------------------------------------ */
/* Philox4x32-10, Salmon, Moraes, Dror, Shaw, "Parallel random numbers: */
/* as easy as 1, 2, 3", SC'11: 10 rounds of the 4x32 S-box with key     */
/* schedule (k0,k1) += (0x9E3779B9, 0xBB67AE85) between rounds.         */
/* ------------------------------------------------------------------ */
void oracle_philox4x32(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int r = 0; r < 10; ++r) {
        if (r > 0) { k0 += 0x9E3779B9u; k1 += 0xBB67AE85u; }
        uint64_t p0 = (uint64_t)0xD2511F53u * (uint64_t)c0;
        uint64_t p1 = (uint64_t)0xCD9E8D57u * (uint64_t)c2;
        uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        uint32_t n0 = hi1 ^ c1 ^ k0, n1 = lo1, n2 = hi0 ^ c3 ^ k1, n3 = lo0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* Slot layout: key = seed, counter = (pos, block, seq, 0).  A 32-bit word
 * w maps to ((w >> 8) + 0.5) * 2^-24, a value strictly inside (0,1) that
 * fp32 and fp64 both hold exactly. */
void oracle_uniforms(uint64_t seed, uint32_t seq, uint32_t pos, uint32_t block, double u[4])
{
    uint32_t ctr[4] = {pos, block, seq, 0u};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t w[4];
    oracle_philox4x32(ctr, key, w);
    for (int i = 0; i < 4; ++i) u[i] = ((double)(w[i] >> 8) + 0.5) * (1.0 / 16777216.0);
}

/* bf16 = 8 significant bits.  Direct nearest-even rounding of the exact value. */
double oracle_round_bf16(double x)
{
    if (x == 0.0 || !isfinite(x)) return x;
    int e;
    double m = frexp(x, &e);          /* x = m 2^e, 0.5 <= |m| < 1 */
    double r = nearbyint(ldexp(m, 8)); /* default mode: ties to even */
    return ldexp(r, e - 8);
}

/* ------------------------------------------------------------------ */
/* Model parameters: the blob layout of include/tppsd.h, read as-is.     */
/* ------------------------------------------------------------------ */
typedef struct {
    const float *w_qkv, *b_qkv, *w_o, *b_o, *ln1_g, *ln1_b, *w_1, *b_1, *w_2, *b_2, *ln2_g, *ln2_b;
} layer_p;

typedef struct {
    int L, d, nh, F, M, K, bf16;
    int enc;                       /* 0 THP, 1 SAHP, 2 AttNHP (App. D.4) */
    const float *type_emb;
    const float *tenc_w;           /* SAHP: per-dimension frequencies w_j [d] */
    double scale_m, scale_M;       /* AttNHP: time scales m, M */
    layer_p layer[64];
    const float *E, *v_w, *b_w, *v_mu, *b_mu, *v_s, *b_s, *v_k1, *b_k1, *v_k2, *b_k2;
} model_t;

/* Blob size of a model: THP and SAHP layers carry QKV, the output
 * projection, two LayerNorms and the FFN; AttNHP layers only QKV over the
 * 2d inputs [z(t); h].  SAHP appends w_j [d], AttNHP its scales (m, M). */
static int64_t model_floats(const int32_t c[8])
{
    int64_t L = c[0], d = c[1], F = c[3], M = c[4], K = c[5], enc = c[7];
    int64_t per_layer = enc == 2 ? 3 * d * 2 * d + 3 * d
                                 : 3 * d * d + 3 * d + d * d + d + 2 * d + F * d + F + d * F + d + 2 * d;
    int64_t tail = enc == 1 ? d : enc == 2 ? 2 : 0;
    return K * d + L * per_layer + 3 * d * d + 3 * (M * d + M) + d * d + d + K * d + K + tail;
}

static int model_init(model_t *m, const int32_t c[8], const float *blob, int64_t n)
{
    if (c[0] < 1 || c[0] > 64 || c[1] < 2 || c[1] > 512 || c[1] % 2 || c[2] < 1 || c[1] % c[2] ||
        c[3] < 1 || c[4] < 1 || c[4] > MAXM || c[5] < 1 || c[5] > MAXK || c[7] < 0 || c[7] > 2)
        return -1;
    if (model_floats(c) != n) return -2;
    m->L = c[0]; m->d = c[1]; m->nh = c[2]; m->F = c[3]; m->M = c[4]; m->K = c[5];
    m->bf16 = c[6] == 1;
    m->enc = c[7];
    m->tenc_w = NULL;
    m->scale_m = m->scale_M = 0.0;
    int d = m->d, F = m->F, M = m->M, K = m->K;
    const float *p = blob;
    m->type_emb = p; p += (int64_t)K * d;
    for (int l = 0; l < m->L; ++l) {
        layer_p *q = &m->layer[l];
        memset(q, 0, sizeof(*q));
        if (m->enc == 2) {
            q->w_qkv = p; p += 3 * d * 2 * d;  q->b_qkv = p; p += 3 * d;
            continue;
        }
        q->w_qkv = p; p += 3 * d * d;  q->b_qkv = p; p += 3 * d;
        q->w_o = p; p += d * d;        q->b_o = p; p += d;
        q->ln1_g = p; p += d;          q->ln1_b = p; p += d;
        q->w_1 = p; p += F * d;        q->b_1 = p; p += F;
        q->w_2 = p; p += d * F;        q->b_2 = p; p += d;
        q->ln2_g = p; p += d;          q->ln2_b = p; p += d;
    }
    m->E = p; p += 3 * d * d;
    m->v_w = p; p += M * d;  m->b_w = p; p += M;
    m->v_mu = p; p += M * d; m->b_mu = p; p += M;
    m->v_s = p; p += M * d;  m->b_s = p; p += M;
    m->v_k1 = p; p += d * d; m->b_k1 = p; p += d;
    m->v_k2 = p; p += K * d; m->b_k2 = p; p += K;
    if (m->enc == 1) { m->tenc_w = p; p += d; }
    if (m->enc == 2) {
        m->scale_m = p[0]; m->scale_M = p[1]; p += 2;
        if (!(m->scale_m > 0.0) || !(m->scale_M > 0.0)) return -1;
    }
    return (p - blob) == n ? 0 : -2;
}

static double rnd(const model_t *m, double x) { return m->bf16 ? oracle_round_bf16(x) : x; }

/* y[o] = sum_i W[o][i] x[i] + b[o]  (W row-major [out][in]) */
static void linear(const float *W, const float *b, const double *x, int in, int out, double *y)
{
    for (int o = 0; o < out; ++o) {
        double acc = 0.0;
        for (int i = 0; i < in; ++i) acc += (double)W[(int64_t)o * in + i] * x[i];
        y[o] = acc + (b ? (double)b[o] : 0.0);
    }
}

static void layer_norm(double *x, int d, const float *g, const float *b)
{
    double mean = 0.0, var = 0.0;
    for (int i = 0; i < d; ++i) mean += x[i];
    mean /= d;
    for (int i = 0; i < d; ++i) var += (x[i] - mean) * (x[i] - mean);
    var /= d;
    double inv = 1.0 / sqrt(var + LN_EPS);
    for (int i = 0; i < d; ++i) x[i] = (x[i] - mean) * inv * (double)g[i] + (double)b[i];
}

static double logsumexp(const double *v, int n)
{
    double mx = v[0];
    for (int i = 1; i < n; ++i) if (v[i] > mx) mx = v[i];
    double s = 0.0;
    for (int i = 0; i < n; ++i) s += exp(v[i] - mx);
    return mx + log(s);
}

/* Temporal encoding, THP form (App. D.4): [z]_j = sin(t / 10000^{j/D}) for
 * even j, cos(t / 10000^{(j-1)/D}) for odd j; t is the absolute time. */
void oracle_temporal_encoding(int32_t d, double t, double *out)
{
    for (int j = 0; j < d; ++j) {
        int je = j - (j & 1);
        double arg = t / pow(10000.0, (double)je / (double)d);
        out[j] = (j & 1) ? cos(arg) : sin(arg);
    }
}

/* Temporal encoding of a model (App. D.4), j 0-based, je = j - (j mod 2):
 *   THP:    sin / cos (t / 10000^{je/D})                 (even / odd j)
 *   SAHP:   sin / cos (j / 10000^{je/D} + w_j t)
 *   AttNHP: sin / cos (t / (m (5M/m)^{je/D}))
 * Readings: the AttNHP formula's "t/m * (5M/m)^{j/D}" is taken as t divided
 * by the wavelength m (5M/m)^{j/D} (wavelengths from m to 5M), and its odd
 * dimensions as cos (the printed sin on both lines would duplicate every
 * pair). */
static void model_temporal_encoding(const model_t *m, double t, double *out)
{
    int d = m->d;
    for (int j = 0; j < d; ++j) {
        int je = j - (j & 1);
        double arg;
        if (m->enc == 1)
            arg = (double)j / pow(10000.0, (double)je / (double)d) + (double)m->tenc_w[j] * t;
        else if (m->enc == 2)
            arg = t / (m->scale_m * pow(5.0 * m->scale_M / m->scale_m, (double)je / (double)d));
        else
            arg = t / pow(10000.0, (double)je / (double)d);
        out[j] = (j & 1) ? cos(arg) : sin(arg);
    }
}

int oracle_model_temporal_encoding(const int32_t cfg[8], const float *blob, int64_t blob_floats,
                                   double t, double *out)
{
    model_t m;
    if (model_init(&m, cfg, blob, blob_floats)) return -1;
    model_temporal_encoding(&m, t, out);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Head of Sec. 4.2.  Row layout [log w | mu | s | log f].               */
/* ------------------------------------------------------------------ */
/* A head of the Poisson draft (App. D.3, history-independent) has
 * poisson = 1, M = 1, v[0] = log lambda and v[3 + k] = log p_k: the
 * inter-event density lambda exp(-lambda tau) and iid marks from p. */
typedef struct { int M, K, poisson; double v[3 * MAXM + MAXK]; } head_t;

static void model_head(const model_t *m, const double *h, head_t *out)
{
    int d = m->d, M = m->M, K = m->K;
    double e[3 * 512], a[512], lw[MAXM], lk[MAXK];
    out->M = M; out->K = K; out->poisson = 0;
    linear(m->E, NULL, h, d, 3 * d, e);                     /* e = E h, split e1|e2|e3 */
    linear(m->v_w, m->b_w, e, d, M, lw);                    /* w = softmax(V_w e1 + b_w) */
    double z = logsumexp(lw, M);
    for (int i = 0; i < M; ++i) out->v[i] = lw[i] - z;
    linear(m->v_mu, m->b_mu, e + d, d, M, out->v + M);      /* mu = V_mu e2 + b_mu */
    linear(m->v_s, m->b_s, e + 2 * d, d, M, out->v + 2 * M); /* sigma = exp(V_s e3 + b_s) */
    linear(m->v_k1, m->b_k1, h, d, d, a);                   /* f = softmax(V2 tanh(V1 h + b1) + b2) */
    for (int i = 0; i < d; ++i) a[i] = tanh(a[i]);
    linear(m->v_k2, m->b_k2, a, d, K, lk);
    z = logsumexp(lk, K);
    for (int i = 0; i < K; ++i) out->v[3 * M + i] = lk[i] - z;
}

/* log g(tau | h): log of the log-normal mixture density of Sec. 4.2,
 * log sum_m w_m (tau sqrt(2 pi) sigma_m)^-1 exp(-(log tau - mu_m)^2 / (2 sigma_m^2)). */
double oracle_log_g(int32_t M, const double *hd, double tau)
{
    double lt = log(tau), c[MAXM];
    for (int m = 0; m < M; ++m) {
        double s = hd[2 * M + m], zz = (lt - hd[M + m]) / exp(s);
        c[m] = hd[m] - lt - s - 0.5 * LOG_2PI - 0.5 * zz * zz;
    }
    return logsumexp(c, M);
}

double oracle_log_f(int32_t M, const double *hd, int32_t k) { return hd[3 * M + k]; }

/* log g of either kind of head: the mixture above, or for the Poisson
 * draft the exponential density, log lambda - lambda tau. */
static double head_log_g(const head_t *h, double tau)
{
    if (h->poisson) return h->v[0] - exp(h->v[0]) * tau;
    return oracle_log_g(h->M, h->v, tau);
}

/* log(1 - Phi(z)) = log(erfc(z / sqrt 2) / 2); for z beyond the range where
 * erfc underflows, the leading term of its asymptotic expansion,
 * erfc(x) ~ exp(-x^2) / (x sqrt(pi)). */
static double log_normal_tail(double z)
{
    double x = z / sqrt(2.0);
    if (x < 25.0) return log(0.5 * erfc(x));
    return -x * x - log(x * 1.7724538509055160273) - log(2.0);  /* sqrt(pi) */
}

/* log S(u) = log(1 - G(u)), G the log-normal mixture CDF of Sec. 4.2:
 * 1 - G(u) = sum_m w_m (1 - Phi((log u - mu_m) / sigma_m)).  This is the
 * survival term of the log-likelihood on [0, T] (Sec. 3.1, Eq. 2): no event
 * in the u = T - t_last after the last one.  u <= 0 gives 0 (log 1). */
double oracle_log_survival(int32_t M, const double *hd, double u)
{
    if (!(u > 0.0)) return 0.0;
    double lu = log(u), c[MAXM];
    for (int m = 0; m < M; ++m) c[m] = hd[m] + log_normal_tail((lu - hd[M + m]) / exp(hd[2 * M + m]));
    return logsumexp(c, M);
}

/* Categorical choice: smallest index whose running sum of p reaches u * sum(p).
 * *margin gets the distance of u * sum to the nearest boundary, / sum. */
static int categorical(const double *p, int n, double u, double *margin)
{
    double tot = 0.0;
    for (int i = 0; i < n; ++i) tot += p[i];
    double target = u * tot, run = 0.0, best = INFINITY;
    int pick = n - 1, found = 0;
    for (int i = 0; i < n; ++i) {
        run += p[i];
        double dist = fabs(run - target);
        if (i < n - 1 && dist < best) best = dist;
        if (!found && run >= target) { pick = i; found = 1; }
    }
    if (margin) *margin = tot > 0 ? best / tot : 0.0;
    return pick;
}

static void upd(double *mg, double v) { if (mg && v < *mg) *mg = v; }

/* Time draw of Sec. 4.2 / App. A.1: z ~ Categorical(w), eps ~ N(0,1) by
 * Box-Muller (cos branch), tau = exp(mu_z + sigma_z eps). */
static double draw_time(const double *hd, int M, double u_comp, double u1, double u2, double *mg)
{
    double w[MAXM], mgc;
    for (int m = 0; m < M; ++m) w[m] = exp(hd[m]);
    int z = categorical(w, M, u_comp, &mgc);
    upd(mg, mgc);
    double eps = sqrt(-2.0 * log(u1)) * cos(TWO_PI * u2);
    return exp(hd[M + z] + exp(hd[2 * M + z]) * eps);
}

static int draw_mark(const double *hd, int M, int K, double u, double *mg)
{
    double f[MAXK], mgc;
    for (int k = 0; k < K; ++k) f[k] = exp(hd[3 * M + k]);
    int k = categorical(f, K, u, &mgc);
    upd(mg, mgc);
    return k;
}

/* Direct sample of the next event from one head with slot block 0:
 * {u_comp, u_bm1, u_bm2, u_mark}.  Reading for the Poisson draft: the
 * time by inversion of the exponential CDF from the first word,
 * tau = -log(u_comp) / lambda; the mark from p with u_mark. */
static void draw_event(const head_t *hd, uint64_t seed, uint32_t seq, uint32_t pos,
                       double *tau, int *k, double *mg)
{
    double u[4];
    oracle_uniforms(seed, seq, pos, 0, u);
    if (hd->poisson) *tau = -log(u[0]) / exp(hd->v[0]);
    else *tau = draw_time(hd->v, hd->M, u[0], u[1], u[2], mg);
    *k = draw_mark(hd->v, hd->M, hd->K, u[3], mg);
}

/* Theorem 1: propose tau ~ g_T, accept iff eps < max(0, g_T - g_D) / g_T.
 * Iteration i uses slot block 2 + i: {u_comp, u_bm1, u_bm2, u_acc}.
 * Reading: capped at RESAMPLE_CAP iterations; on the cap the last proposal
 * is returned and *cap_hit set. */
static double resample_time(const head_t *hT, const head_t *hD, uint64_t seed,
                            uint32_t seq, uint32_t pos, int *iters, int *cap_hit, double *mg)
{
    double tau = 1.0;
    for (int i = 0; i < RESAMPLE_CAP; ++i) {
        double u[4];
        oracle_uniforms(seed, seq, pos, 2u + (uint32_t)i, u);
        tau = draw_time(hT->v, hT->M, u[0], u[1], u[2], mg);
        double lgT = oracle_log_g(hT->M, hT->v, tau), lgD = head_log_g(hD, tau);
        double alpha = 1.0 - exp(lgD - lgT);       /* (g_T - g_D) / g_T */
        if (alpha < 0.0) alpha = 0.0;
        upd(mg, fabs(u[3] - alpha));
        if (u[3] < alpha) { if (iters) *iters = i + 1; return tau; }
    }
    if (iters) *iters = RESAMPLE_CAP;
    if (cap_hit) *cap_hit = 1;
    return tau;
}

/* Eq. 4: f' = norm(max(0, f_T - f_D)), drawn with u.  Reading: if the
 * residual mass is below 1e-12 (a rejection of numerically zero
 * probability) the mark is drawn from f_T instead. */
static int resample_mark(int MT, const double *hT, int MD, const double *hD, int K, double u, double *mg)
{
    double r[MAXK], tot = 0.0, mgc;
    for (int k = 0; k < K; ++k) {
        double v = exp(hT[3 * MT + k]) - exp(hD[3 * MD + k]);
        r[k] = v > 0.0 ? v : 0.0;
        tot += r[k];
    }
    if (tot < 1e-12) return draw_mark(hT, MT, K, u, mg);
    int k = categorical(r, K, u, &mgc);
    upd(mg, mgc);
    return k;
}

/* ------------------------------------------------------------------ */
/* Models behind one interface: step(event) appends an event at position */
/* len() and returns the head that predicts the next event.              */
/* ------------------------------------------------------------------ */
typedef struct model_ops {
    int (*len)(void *st);
    void (*step)(void *st, double t, int k, head_t *out);
    void (*truncate)(void *st, int n);
} model_ops;

/* Transformer TPP of Sec. 4.2.  Encoder: X = Z + K W (sum fusion), then
 * causal Transformer layers.  Reading (the paper fixes only attention +
 * residual, App. D.4): post-LN layers h <- LN(h + MHA(h)),
 * h <- LN(h + W2 ReLU(W1 h + b1) + b2); softmax attention with scale
 * 1/sqrt(d_head); LayerNorm eps 1e-5; no final LayerNorm. */
typedef struct {
    const model_t *m;
    int n, cap, recompute;
    double *K, *V;          /* [L][cap][d] */
    double *ev_t;           /* recompute mode: events so far */
    int *ev_k;
} tstate;

static void tstate_init(tstate *s, const model_t *m, int cap, int recompute)
{
    s->m = m; s->n = 0; s->cap = cap; s->recompute = recompute;
    s->K = (double *)malloc(sizeof(double) * (size_t)m->L * cap * m->d);
    s->V = (double *)malloc(sizeof(double) * (size_t)m->L * cap * m->d);
    s->ev_t = (double *)malloc(sizeof(double) * cap);
    s->ev_k = (int *)malloc(sizeof(int) * cap);
}

static void tstate_free(tstate *s) { free(s->K); free(s->V); free(s->ev_t); free(s->ev_k); }

/* Encode the event at position pos (= number of cached positions) and
 * leave its final-layer hidden state in h. */
static void encode_position(tstate *s, int pos, double t, int k, double *h)
{
    const model_t *m = s->m;
    int d = m->d, nh = m->nh, dh = d / nh, F = m->F;
    double xin[512], qkv[3 * 512], att[512], tmp[512], *hid;
    hid = (double *)malloc(sizeof(double) * F * 2);
    double *hin = hid + F;
    double z[512], u[1024];
    model_temporal_encoding(m, t, z);
    for (int i = 0; i < d; ++i) h[i] = z[i] + (double)m->type_emb[(int64_t)k * d + i];
    double scale = 1.0 / sqrt((double)dh);
    double *sc = (double *)malloc(sizeof(double) * (pos + 1));
    if (m->enc == 2) {
        /* AttNHP layer (App. D.4): q, k, v = W [1; z(t); h] (the 1 is the
         * bias), per head a = sum_j f_j v_j / (1 + sum_j f_j) with
         * f_j = exp(q k_j / sqrt(d_head)) over keys j <= pos, then
         * h <- h + tanh(a) (heads concatenated; no output projection,
         * LayerNorm or FFN).  bf16 rounding at the GEMM input [z; h] and of
         * q, k, v. */
        for (int l = 0; l < m->L; ++l) {
            const layer_p *P = &m->layer[l];
            double *Kl = s->K + (size_t)l * s->cap * d, *Vl = s->V + (size_t)l * s->cap * d;
            for (int i = 0; i < d; ++i) { u[i] = rnd(m, z[i]); u[d + i] = rnd(m, h[i]); }
            linear(P->w_qkv, P->b_qkv, u, 2 * d, 3 * d, qkv);
            for (int i = 0; i < 3 * d; ++i) qkv[i] = rnd(m, qkv[i]);
            memcpy(Kl + (size_t)pos * d, qkv + d, sizeof(double) * d);
            memcpy(Vl + (size_t)pos * d, qkv + 2 * d, sizeof(double) * d);
            for (int hh = 0; hh < nh; ++hh) {
                const double *q = qkv + hh * dh;
                double mx = 0.0;                    /* the "1" term: exp(0) */
                for (int j = 0; j <= pos; ++j) {
                    double a = 0.0;
                    for (int c = 0; c < dh; ++c) a += q[c] * Kl[(size_t)j * d + hh * dh + c];
                    sc[j] = a * scale;
                    if (sc[j] > mx) mx = sc[j];
                }
                double den = exp(-mx);
                for (int j = 0; j <= pos; ++j) { sc[j] = exp(sc[j] - mx); den += sc[j]; }
                for (int c = 0; c < dh; ++c) {
                    double a = 0.0;
                    for (int j = 0; j <= pos; ++j) a += sc[j] * Vl[(size_t)j * d + hh * dh + c];
                    att[hh * dh + c] = a / den;
                }
            }
            for (int i = 0; i < d; ++i) h[i] += tanh(att[i]);
        }
        free(sc);
        free(hid);
        return;
    }
    for (int l = 0; l < m->L; ++l) {
        const layer_p *P = &m->layer[l];
        double *Kl = s->K + (size_t)l * s->cap * d, *Vl = s->V + (size_t)l * s->cap * d;
        for (int i = 0; i < d; ++i) xin[i] = rnd(m, h[i]);
        linear(P->w_qkv, P->b_qkv, xin, d, 3 * d, qkv);
        for (int i = 0; i < 3 * d; ++i) qkv[i] = rnd(m, qkv[i]);
        memcpy(Kl + (size_t)pos * d, qkv + d, sizeof(double) * d);
        memcpy(Vl + (size_t)pos * d, qkv + 2 * d, sizeof(double) * d);
        for (int hh = 0; hh < nh; ++hh) {            /* causal softmax attention, keys 0..pos */
            const double *q = qkv + hh * dh;
            double mx = -INFINITY;
            for (int j = 0; j <= pos; ++j) {
                double a = 0.0;
                for (int c = 0; c < dh; ++c) a += q[c] * Kl[(size_t)j * d + hh * dh + c];
                sc[j] = a * scale;
                if (sc[j] > mx) mx = sc[j];
            }
            double den = 0.0;
            for (int j = 0; j <= pos; ++j) { sc[j] = exp(sc[j] - mx); den += sc[j]; }
            for (int c = 0; c < dh; ++c) {
                double a = 0.0;
                for (int j = 0; j <= pos; ++j) a += sc[j] * Vl[(size_t)j * d + hh * dh + c];
                att[hh * dh + c] = a / den;
            }
        }
        for (int i = 0; i < d; ++i) xin[i] = rnd(m, att[i]);
        linear(P->w_o, P->b_o, xin, d, d, tmp);
        for (int i = 0; i < d; ++i) h[i] += tmp[i];
        layer_norm(h, d, P->ln1_g, P->ln1_b);
        for (int i = 0; i < d; ++i) xin[i] = rnd(m, h[i]);
        linear(P->w_1, P->b_1, xin, d, F, hid);
        for (int i = 0; i < F; ++i) hin[i] = rnd(m, hid[i] > 0.0 ? hid[i] : 0.0);
        linear(P->w_2, P->b_2, hin, F, d, tmp);
        for (int i = 0; i < d; ++i) h[i] += tmp[i];
        layer_norm(h, d, P->ln2_g, P->ln2_b);
    }
    free(sc);
    free(hid);
}

static int t_len(void *st) { return ((tstate *)st)->n; }

static void t_step(void *st, double t, int k, head_t *out)
{
    tstate *s = (tstate *)st;
    double h[512];
    int pos = s->n;
    s->ev_t[pos] = t; s->ev_k[pos] = k;
    if (s->recompute) {
        /* No cache: encode every position 0..pos again from the events. */
        for (int p = 0; p <= pos; ++p) encode_position(s, p, s->ev_t[p], s->ev_k[p], h);
    } else {
        encode_position(s, pos, t, k, h);
    }
    s->n = pos + 1;
    model_head(s->m, h, out);
}

static void t_truncate(void *st, int n) { tstate *s = (tstate *)st; if (n < s->n) s->n = n; }

static const model_ops TRANSFORMER_OPS = {t_len, t_step, t_truncate};

/* Toy model: the head for the next event is table[previous mark]. */
typedef struct { int M, K, n; const double *table; } toystate;
static int toy_len(void *st) { return ((toystate *)st)->n; }
static void toy_step(void *st, double t, int k, head_t *out)
{
    toystate *s = (toystate *)st;
    (void)t;
    out->M = s->M; out->K = s->K; out->poisson = 0;
    memcpy(out->v, s->table + (size_t)k * (3 * s->M + s->K), sizeof(double) * (3 * s->M + s->K));
    s->n++;
}
static void toy_truncate(void *st, int n) { toystate *s = (toystate *)st; if (n < s->n) s->n = n; }
static const model_ops TOY_OPS = {toy_len, toy_step, toy_truncate};

/* Poisson draft (App. D.3): the same head after every event. */
typedef struct { int n; head_t head; } poisstate;
static int pois_len(void *st) { return ((poisstate *)st)->n; }
static void pois_step(void *st, double t, int k, head_t *out)
{
    poisstate *s = (poisstate *)st;
    (void)t; (void)k;
    *out = s->head;
    s->n++;
}
static void pois_truncate(void *st, int n) { poisstate *s = (poisstate *)st; if (n < s->n) s->n = n; }
static const model_ops POISSON_OPS = {pois_len, pois_step, pois_truncate};

/* Head of the Poisson draft from the rate and the mark probabilities
 * (normalised here).  Returns -1 unless lambda > 0, p_k >= 0, sum p > 0. */
static int poisson_head(double lambda, const double *p, int K, head_t *h)
{
    if (!(lambda > 0.0) || !isfinite(lambda) || K < 1 || K > MAXK) return -1;
    double tot = 0.0;
    for (int k = 0; k < K; ++k) {
        if (!(p[k] >= 0.0) || !isfinite(p[k])) return -1;
        tot += p[k];
    }
    if (!(tot > 0.0)) return -1;
    h->M = 1; h->K = K; h->poisson = 1;
    h->v[0] = log(lambda); h->v[1] = 0.0; h->v[2] = 0.0;
    for (int k = 0; k < K; ++k) h->v[3 + k] = log(p[k] / tot);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Samplers over one sequence.  ev_* hold history + generated events at  */
/* absolute indices; H history events, N to generate.                    */
/* ------------------------------------------------------------------ */
typedef struct { double *tau, *t; int *k; double *mg; } evbuf;

/* Naive autoregressive sampling, Sec. 4.2: sample, append, repeat. */
/* Stop rule (Alg. 1): a sequence ends once its last event lies beyond the
 * end time t_end, or after N generated events; the result is the events
 * with t <= t_end (a prefix, since times increase).  t_end = +inf gives the
 * fixed-count form.  Returns the number of generated events kept. */
static int kept_events(const evbuf *ev, int H, int n, int N, double t_end)
{
    int c = n - H < N ? n - H : N;
    while (c > 0 && ev->t[H + c - 1] > t_end) --c;
    return c;
}

/* Naive autoregressive sampling, Sec. 4.2: sample, append, repeat. */
static int ar_sequence(const model_ops *T, void *ts, evbuf *ev, int H, int N, double t_end,
                       uint64_t seed, uint32_t seq)
{
    head_t hd;
    for (int p = 0; p < H - 1; ++p) T->step(ts, ev->t[p], ev->k[p], &hd);
    int n = H;
    for (int p = H; p < H + N && ev->t[p - 1] <= t_end; ++p) {
        T->step(ts, ev->t[p - 1], ev->k[p - 1], &hd);   /* head after event p-1 */
        double tau;
        int k;
        draw_event(&hd, seed, seq, (uint32_t)p, &tau, &k, &ev->mg[p]);
        ev->tau[p] = tau; ev->t[p] = ev->t[p - 1] + tau; ev->k[p] = k;
        n = p + 1;
    }
    return kept_events(ev, H, n, N, t_end);
}

/* TPP-SD, Sec. 4.3 and Alg. 1, with these readings:
 *  - L = first draft position where the time OR the mark test fails, else
 *    gamma + 1; resampling happens iff L <= gamma (Alg. 1's "L < gamma" and
 *    its minimum over an empty set are read this way).
 *  - both tests are taken at every position with their own uniforms; at L
 *    only the failing component(s) are redrawn: tau from g' (Theorem 1),
 *    k from f' (Eq. 4); a passing component is kept (redrawing it from g'
 *    would give law g' != g_T, App. A.2).
 *  - after a fully accepted draft one bonus event is drawn from the target
 *    head that follows the last draft (the LLM rule of Sec. 2.3), unless
 *    FLAG_NO_BONUS.
 *  - stop once the last emitted event lies beyond t_end (Alg. 1's end
 *    time) or after N generated events; keep the events with t <= t_end.
 * Cache invariant at round start: T has encoded all events but the last;
 * D has encoded all but the last one or two.  Returns the kept count. */
static int sd_sequence(const model_ops *T, void *ts, const model_ops *D, void *ds,
                       evbuf *ev, int H, int N, double t_end, int gamma, uint64_t seed, uint32_t seq,
                       uint32_t flags, int64_t *st)
{
    head_t hd, dhead[64 + 1], thead[64 + 1];
    double tau_hat[64 + 1];
    int k_hat[64 + 1];
    for (int p = 0; p < H - 1; ++p) { T->step(ts, ev->t[p], ev->k[p], &hd); D->step(ds, ev->t[p], ev->k[p], &hd); }
    int n = H;                                      /* events so far */
    while (n < H + N && ev->t[n - 1] <= t_end) {
        /* Drafting: gamma events from M_D, recording their heads. */
        for (int p = D->len(ds); p <= n - 1; ++p) D->step(ds, ev->t[p], ev->k[p], &hd);
        for (int l = 1; l <= gamma; ++l) {
            int p = n + l - 1;
            dhead[l] = hd;
            draw_event(&hd, seed, seq, (uint32_t)p, &tau_hat[l], &k_hat[l], &ev->mg[p]);
            ev->tau[p] = tau_hat[l]; ev->t[p] = ev->t[p - 1] + tau_hat[l]; ev->k[p] = k_hat[l];
            if (l < gamma) D->step(ds, ev->t[p], ev->k[p], &hd);
        }
        /* Verification: M_T over positions n-1 .. n+gamma-1 (gamma+1 heads). */
        for (int lp = 0; lp <= gamma; ++lp) T->step(ts, ev->t[n - 1 + lp], ev->k[n - 1 + lp], &thead[lp]);
        /* Tests: eps^tau < g_T/g_D, eps^k < f_T/f_D, first failure L. */
        int L = gamma + 1, acc_tau = 1, acc_k = 1;
        double u[4];
        for (int l = 1; l <= gamma; ++l) {
            int p = n + l - 1;
            const double *hT = thead[l - 1].v, *hD = dhead[l].v;
            int M_T = thead[l - 1].M, M_D = dhead[l].M;
            oracle_uniforms(seed, seq, (uint32_t)p, 1, u);
            double rt = exp(oracle_log_g(M_T, hT, tau_hat[l]) - head_log_g(&dhead[l], tau_hat[l]));
            double rk = exp(oracle_log_f(M_T, hT, k_hat[l]) - oracle_log_f(M_D, hD, k_hat[l]));
            if (rt > 1.0) rt = 1.0;
            if (rk > 1.0) rk = 1.0;
            acc_tau = u[0] < rt;
            acc_k = u[1] < rk;
            upd(&ev->mg[p], fabs(u[0] - rt));
            upd(&ev->mg[p], fabs(u[1] - rk));
            if (!acc_tau || !acc_k) { L = l; break; }
        }
        int A = L - 1, emitted;
        st[0] += 1; st[1] += gamma; st[2] += A;
        if (L <= gamma) {
            int p = n + L - 1;
            double tau = tau_hat[L];
            int k = k_hat[L];
            const head_t *hT = &thead[L - 1], *hD = &dhead[L];
            if (!acc_tau) {
                int it = 0, cap = 0;
                tau = resample_time(hT, hD, seed, seq, (uint32_t)p, &it, &cap, &ev->mg[p]);
                st[3] += it; st[4] += cap;
            }
            if (!acc_k) k = resample_mark(hT->M, hT->v, hD->M, hD->v, hT->K, u[2], &ev->mg[p]);
            ev->tau[p] = tau; ev->t[p] = ev->t[p - 1] + tau; ev->k[p] = k;
            emitted = L;
        } else if (!(flags & FLAG_NO_BONUS)) {
            int p = n + gamma;
            double tau;
            int k;
            draw_event(&thead[gamma], seed, seq, (uint32_t)p, &tau, &k, &ev->mg[p]);
            ev->tau[p] = tau; ev->t[p] = ev->t[p - 1] + tau; ev->k[p] = k;
            emitted = gamma + 1;
        } else {
            emitted = gamma;
        }
        /* Roll back: T keeps all emitted events but the last; D keeps what
         * it encoded of the accepted prefix. */
        int n_new = n + emitted;
        T->truncate(ts, n_new - 1);
        int keepD = n + A;
        if (D->len(ds) > keepD) D->truncate(ds, keepD);
        n = n_new;
    }
    return kept_events(ev, H, n, N, t_end);
}

/* ------------------------------------------------------------------ */
/* Batch entry points                                                    */
/* ------------------------------------------------------------------ */
static int nthreads_or_default(int n)
{
#ifdef _OPENMP
    return n > 0 ? n : omp_get_max_threads();
#else
    (void)n;
    return 1;
#endif
}

static void load_history(evbuf *ev, const float *tau, const int32_t *k, int H)
{
    double t = 0.0;                                 /* t_0 = 0, t_i = t_{i-1} + tau_i */
    for (int p = 0; p < H; ++p) {
        t += (double)tau[p];
        ev->tau[p] = tau[p]; ev->t[p] = t; ev->k[p] = k[p]; ev->mg[p] = INFINITY;
    }
}

static void evbuf_alloc(evbuf *ev, int cap)
{
    ev->tau = (double *)malloc(sizeof(double) * cap);
    ev->t = (double *)malloc(sizeof(double) * cap);
    ev->k = (int *)malloc(sizeof(int) * cap);
    ev->mg = (double *)malloc(sizeof(double) * cap);
    for (int i = 0; i < cap; ++i) ev->mg[i] = INFINITY;
}

static void evbuf_free(evbuf *ev) { free(ev->tau); free(ev->t); free(ev->k); free(ev->mg); }

/* The first c generated events of sequence b; slots c..N-1 get NaN / -1. */
static void store_out(const evbuf *ev, int H, int N, int c, int64_t b, double *o_tau, double *o_t,
                      int32_t *o_k, double *o_mg)
{
    for (int i = 0; i < N; ++i) {
        const int in = i < c;
        if (o_tau) o_tau[b * N + i] = in ? ev->tau[H + i] : NAN;
        if (o_t) o_t[b * N + i] = in ? ev->t[H + i] : NAN;
        if (o_k) o_k[b * N + i] = in ? ev->k[H + i] : -1;
        if (o_mg) o_mg[b * N + i] = in ? ev->mg[H + i] : NAN;
    }
}

int oracle_sample_ar_until(const int32_t cfgT[8], const float *blobT, int64_t nT,
                           int32_t B, int32_t H, const float *hist_tau, const int32_t *hist_marks,
                           int32_t N, double t_end, uint64_t seed, int32_t recompute,
                           const int32_t *seq_ids, double *out_tau, double *out_t, int32_t *out_k,
                           double *out_margin, int32_t *out_count, int32_t nthreads)
{
    model_t mT;
    if (model_init(&mT, cfgT, blobT, nT)) return -1;
    if (B < 0 || H < 1 || N < 0) return -1;
    int cap = H + N + 1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads_or_default(nthreads))
    for (int b = 0; b < B; ++b) {
        evbuf ev;
        tstate ts;
        evbuf_alloc(&ev, cap);
        tstate_init(&ts, &mT, cap, recompute);
        load_history(&ev, hist_tau + (int64_t)b * H, hist_marks + (int64_t)b * H, H);
        const int c = ar_sequence(&TRANSFORMER_OPS, &ts, &ev, H, N, t_end, seed,
                                  (uint32_t)(seq_ids ? seq_ids[b] : b));
        store_out(&ev, H, N, c, b, out_tau, out_t, out_k, out_margin);
        if (out_count) out_count[b] = c;
        tstate_free(&ts);
        evbuf_free(&ev);
    }
    return 0;
}

int oracle_sample_sd_until(const int32_t cfgT[8], const float *blobT, int64_t nT,
                           const int32_t cfgD[8], const float *blobD, int64_t nD,
                           int32_t B, int32_t H, const float *hist_tau, const int32_t *hist_marks,
                           int32_t N, double t_end, int32_t gamma, uint64_t seed, uint32_t flags,
                           int32_t recompute, const int32_t *seq_ids,
                           double *out_tau, double *out_t, int32_t *out_k, double *out_margin,
                           int32_t *out_count, int64_t *stats, int32_t nthreads)
{
    model_t mT, mD;
    if (model_init(&mT, cfgT, blobT, nT) || model_init(&mD, cfgD, blobD, nD)) return -1;
    if (mT.K != mD.K || gamma < 1 || gamma > 64 || B < 0 || H < 1 || N < 0) return -1;
    int cap = H + N + gamma + 2;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads_or_default(nthreads))
    for (int b = 0; b < B; ++b) {
        evbuf ev;
        tstate ts, ds;
        int64_t st[5] = {0, 0, 0, 0, 0};
        evbuf_alloc(&ev, cap);
        tstate_init(&ts, &mT, cap, recompute);
        tstate_init(&ds, &mD, cap, recompute);
        load_history(&ev, hist_tau + (int64_t)b * H, hist_marks + (int64_t)b * H, H);
        const int c = sd_sequence(&TRANSFORMER_OPS, &ts, &TRANSFORMER_OPS, &ds, &ev, H, N, t_end, gamma,
                                  seed, (uint32_t)(seq_ids ? seq_ids[b] : b), flags, st);
        store_out(&ev, H, N, c, b, out_tau, out_t, out_k, out_margin);
        if (out_count) out_count[b] = c;
        if (stats) for (int i = 0; i < 5; ++i) stats[(int64_t)b * 5 + i] = st[i];
        tstate_free(&ts);
        tstate_free(&ds);
        evbuf_free(&ev);
    }
    return 0;
}

/* TPP-SD with the Poisson draft of App. D.3 (rate lambda, mark
 * probabilities p[K]) in place of the draft Transformer. */
int oracle_sample_sd_poisson_until(const int32_t cfgT[8], const float *blobT, int64_t nT,
                                   int32_t B, int32_t H, const float *hist_tau,
                                   const int32_t *hist_marks, int32_t N, double t_end,
                                   int32_t gamma, double lambda, const double *p_marks,
                                   uint64_t seed, uint32_t flags, int32_t recompute,
                                   const int32_t *seq_ids, double *out_tau, double *out_t,
                                   int32_t *out_k, double *out_margin, int32_t *out_count,
                                   int64_t *stats, int32_t nthreads)
{
    model_t mT;
    head_t hp;
    if (model_init(&mT, cfgT, blobT, nT)) return -1;
    if (poisson_head(lambda, p_marks, mT.K, &hp)) return -1;
    if (gamma < 1 || gamma > 64 || B < 0 || H < 1 || N < 0) return -1;
    int cap = H + N + gamma + 2;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads_or_default(nthreads))
    for (int b = 0; b < B; ++b) {
        evbuf ev;
        tstate ts;
        poisstate ds = {0, hp};
        int64_t st[5] = {0, 0, 0, 0, 0};
        evbuf_alloc(&ev, cap);
        tstate_init(&ts, &mT, cap, recompute);
        load_history(&ev, hist_tau + (int64_t)b * H, hist_marks + (int64_t)b * H, H);
        const int c = sd_sequence(&TRANSFORMER_OPS, &ts, &POISSON_OPS, &ds, &ev, H, N, t_end, gamma,
                                  seed, (uint32_t)(seq_ids ? seq_ids[b] : b), flags, st);
        store_out(&ev, H, N, c, b, out_tau, out_t, out_k, out_margin);
        if (out_count) out_count[b] = c;
        if (stats) for (int i = 0; i < 5; ++i) stats[(int64_t)b * 5 + i] = st[i];
        tstate_free(&ts);
        evbuf_free(&ev);
    }
    return 0;
}

int oracle_sample_ar(const int32_t cfgT[8], const float *blobT, int64_t nT,
                     int32_t B, int32_t H, const float *hist_tau, const int32_t *hist_marks,
                     int32_t N, uint64_t seed, int32_t recompute, const int32_t *seq_ids,
                     double *out_tau, double *out_t, int32_t *out_k, double *out_margin,
                     int32_t nthreads)
{
    return oracle_sample_ar_until(cfgT, blobT, nT, B, H, hist_tau, hist_marks, N, INFINITY, seed,
                                  recompute, seq_ids, out_tau, out_t, out_k, out_margin, NULL, nthreads);
}

int oracle_sample_sd(const int32_t cfgT[8], const float *blobT, int64_t nT,
                     const int32_t cfgD[8], const float *blobD, int64_t nD,
                     int32_t B, int32_t H, const float *hist_tau, const int32_t *hist_marks,
                     int32_t N, int32_t gamma, uint64_t seed, uint32_t flags, int32_t recompute,
                     const int32_t *seq_ids,
                     double *out_tau, double *out_t, int32_t *out_k, double *out_margin,
                     int64_t *stats, int32_t nthreads)
{
    return oracle_sample_sd_until(cfgT, blobT, nT, cfgD, blobD, nD, B, H, hist_tau, hist_marks, N,
                                  INFINITY, gamma, seed, flags, recompute, seq_ids, out_tau, out_t,
                                  out_k, out_margin, NULL, stats, nthreads);
}

/* Survival term of the log-likelihood on [0, t_end] (Sec. 3.1, Eq. 2) of
 * each sequence's len events: log S(t_end - t_{len-1} | h_{len-1}) from the
 * head after the last event. */
int oracle_score_survival(const int32_t cfg[8], const float *blob, int64_t blob_floats,
                          int32_t B, int32_t len, const float *tau, const int32_t *marks,
                          double t_end, double *out_logS, int32_t recompute, int32_t nthreads)
{
    model_t m;
    if (model_init(&m, cfg, blob, blob_floats)) return -1;
    if (B < 0 || len < 1) return -1;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads_or_default(nthreads))
    for (int b = 0; b < B; ++b) {
        tstate ts;
        head_t hd;
        evbuf ev;
        evbuf_alloc(&ev, len);
        tstate_init(&ts, &m, len, recompute);
        load_history(&ev, tau + (int64_t)b * len, marks + (int64_t)b * len, len);
        for (int i = 0; i < len; ++i) t_step(&ts, ev.t[i], ev.k[i], &hd);
        out_logS[b] = oracle_log_survival(m.M, hd.v, t_end - ev.t[len - 1]);
        tstate_free(&ts);
        evbuf_free(&ev);
    }
    return 0;
}

int oracle_score(const int32_t cfg[8], const float *blob, int64_t blob_floats,
                 int32_t B, int32_t len, const float *tau, const int32_t *marks,
                 double *out_heads, double *out_logg, double *out_logf,
                 int32_t recompute, int32_t nthreads)
{
    model_t m;
    if (model_init(&m, cfg, blob, blob_floats)) return -1;
    if (B < 0 || len < 1) return -1;
    int R = 3 * m.M + m.K;
#pragma omp parallel for schedule(dynamic, 1) num_threads(nthreads_or_default(nthreads))
    for (int b = 0; b < B; ++b) {
        tstate ts;
        head_t hd;
        evbuf ev;
        evbuf_alloc(&ev, len);
        tstate_init(&ts, &m, len, recompute);
        load_history(&ev, tau + (int64_t)b * len, marks + (int64_t)b * len, len);
        if (out_logg) out_logg[(int64_t)b * len] = NAN;
        if (out_logf) out_logf[(int64_t)b * len] = NAN;
        for (int i = 0; i + 1 < len; ++i) {
            t_step(&ts, ev.t[i], ev.k[i], &hd);
            if (out_heads) memcpy(out_heads + ((int64_t)b * len + i) * R, hd.v, sizeof(double) * R);
            if (out_logg) out_logg[(int64_t)b * len + i + 1] = oracle_log_g(m.M, hd.v, ev.tau[i + 1]);
            if (out_logf) out_logf[(int64_t)b * len + i + 1] = oracle_log_f(m.M, hd.v, ev.k[i + 1]);
        }
        tstate_free(&ts);
        evbuf_free(&ev);
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Pieces on fixed heads                                                 */
/* ------------------------------------------------------------------ */
void oracle_sample_head(int32_t M, int32_t K, const double *head, int32_t n, uint64_t seed,
                        double *out_tau, int32_t *out_k)
{
    head_t hd;
    hd.M = M; hd.K = K; hd.poisson = 0;
    memcpy(hd.v, head, sizeof(double) * (3 * M + K));
    for (int i = 0; i < n; ++i) {
        int k;
        draw_event(&hd, seed, 0, (uint32_t)i, &out_tau[i], &k, NULL);
        if (out_k) out_k[i] = k;
    }
}

void oracle_resample_time(int32_t M, const double *headT, const double *headD, int32_t n,
                          uint64_t seed, double *out_tau, int32_t *iters)
{
    head_t hT, hD;
    hT.M = hD.M = M; hT.K = hD.K = 0; hT.poisson = hD.poisson = 0;
    memcpy(hT.v, headT, sizeof(double) * 3 * M);
    memcpy(hD.v, headD, sizeof(double) * 3 * M);
    for (int i = 0; i < n; ++i) {
        int it = 0, cap = 0;
        out_tau[i] = resample_time(&hT, &hD, seed, 0, (uint32_t)i, &it, &cap, NULL);
        if (iters) iters[i] = it;
    }
}

int oracle_resample_time_poisson(int32_t M, const double *headT, double lambda, int32_t n,
                                 uint64_t seed, double *out_tau, int32_t *iters)
{
    head_t hT, hD;
    double one = 1.0;
    if (M < 1 || M > MAXM || poisson_head(lambda, &one, 1, &hD)) return -1;
    hT.M = M; hT.K = 0; hT.poisson = 0;
    memcpy(hT.v, headT, sizeof(double) * 3 * M);
    for (int i = 0; i < n; ++i) {
        int it = 0, cap = 0;
        out_tau[i] = resample_time(&hT, &hD, seed, 0, (uint32_t)i, &it, &cap, NULL);
        if (iters) iters[i] = it;
    }
    return 0;
}

int oracle_sample_poisson(double lambda, int32_t K, const double *p, int32_t n, uint64_t seed,
                          double *out_tau, int32_t *out_k)
{
    head_t hd;
    if (poisson_head(lambda, p, K, &hd)) return -1;
    for (int i = 0; i < n; ++i) {
        int k;
        draw_event(&hd, seed, 0, (uint32_t)i, &out_tau[i], &k, NULL);
        if (out_k) out_k[i] = k;
    }
    return 0;
}

void oracle_resample_mark(int32_t M, int32_t K, const double *headT, const double *headD,
                          int32_t n, uint64_t seed, int32_t *out_k)
{
    for (int i = 0; i < n; ++i) {
        double u[4];
        oracle_uniforms(seed, 0, (uint32_t)i, 1, u);
        out_k[i] = resample_mark(M, headT, M, headD, K, u[2], NULL);
    }
}

int oracle_toy_sd(int32_t M, int32_t K, const double *tableT, const double *tableD,
                  int32_t B, int32_t N, int32_t gamma, uint64_t seed, uint32_t flags,
                  double *out_tau, int32_t *out_k, int64_t *stats)
{
    if (M < 1 || M > MAXM || K < 1 || K > MAXK || gamma < 1 || gamma > 64) return -1;
    int cap = 1 + N + gamma + 2;
    for (int b = 0; b < B; ++b) {
        toystate ts = {M, K, 0, tableT}, ds = {M, K, 0, tableD};
        evbuf ev;
        int64_t st[5] = {0, 0, 0, 0, 0};
        evbuf_alloc(&ev, cap);
        ev.tau[0] = 1.0; ev.t[0] = 1.0; ev.k[0] = 0;
        sd_sequence(&TOY_OPS, &ts, &TOY_OPS, &ds, &ev, 1, N, INFINITY, gamma, seed, (uint32_t)b, flags, st);
        store_out(&ev, 1, N, N, b, out_tau, NULL, out_k, NULL);
        if (stats) for (int i = 0; i < 5; ++i) stats[(int64_t)b * 5 + i] = st[i];
        evbuf_free(&ev);
    }
    return 0;
}

int oracle_toy_sd_poisson(int32_t M, int32_t K, const double *tableT, double lambda,
                          const double *p_marks, int32_t B, int32_t N, int32_t gamma, uint64_t seed,
                          uint32_t flags, double *out_tau, int32_t *out_k, int64_t *stats)
{
    head_t hp;
    if (M < 1 || M > MAXM || gamma < 1 || gamma > 64 || poisson_head(lambda, p_marks, K, &hp)) return -1;
    int cap = 1 + N + gamma + 2;
    for (int b = 0; b < B; ++b) {
        toystate ts = {M, K, 0, tableT};
        poisstate ds = {0, hp};
        evbuf ev;
        int64_t st[5] = {0, 0, 0, 0, 0};
        evbuf_alloc(&ev, cap);
        ev.tau[0] = 1.0; ev.t[0] = 1.0; ev.k[0] = 0;
        sd_sequence(&TOY_OPS, &ts, &POISSON_OPS, &ds, &ev, 1, N, INFINITY, gamma, seed, (uint32_t)b, flags, st);
        store_out(&ev, 1, N, N, b, out_tau, NULL, out_k, NULL);
        if (stats) for (int i = 0; i < 5; ++i) stats[(int64_t)b * 5 + i] = st[i];
        evbuf_free(&ev);
    }
    return 0;
}

int oracle_toy_ar(int32_t M, int32_t K, const double *tableT, int32_t B, int32_t N,
                  uint64_t seed, double *out_tau, int32_t *out_k)
{
    if (M < 1 || M > MAXM || K < 1 || K > MAXK) return -1;
    for (int b = 0; b < B; ++b) {
        toystate ts = {M, K, 0, tableT};
        evbuf ev;
        evbuf_alloc(&ev, 1 + N + 1);
        ev.tau[0] = 1.0; ev.t[0] = 1.0; ev.k[0] = 0;
        ar_sequence(&TOY_OPS, &ts, &ev, 1, N, INFINITY, seed, (uint32_t)b);
        store_out(&ev, 1, N, N, b, out_tau, NULL, out_k, NULL);
        evbuf_free(&ev);
    }
    return 0;
}
