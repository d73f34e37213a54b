// Internal interface between the C-ABI layer (api.cu) and the kernels
// (kernels.cu): device model descriptors, per-call parameters, launchers.
#pragma once
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace tppsd {

// Kernels of a sampling round are launched with programmatic stream
// serialization (each calls pdl_wait() before touching global memory), so a
// kernel's launch overlaps the previous kernel's last CTAs.  g_pdl = 0
// launches them plainly.
extern int g_pdl;
template <typename... P, typename... A>
inline cudaError_t launch_k(void (*k)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, A... args) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = g_pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k, args...);
}

constexpr int MAX_LAYERS = 16;
constexpr int MAX_MIX = 64;
constexpr int MAX_MARKS = 256;
constexpr int MAX_D = 512;

struct LayerW {
    const void* w_qkv; const float* b_qkv;   // [3d][d] storage type, [3d]
    const void* w_o;   const float* b_o;     // [d][d], [d]
    const float* ln1_g; const float* ln1_b;  // [d]
    const void* w_1;   const float* b_1;     // [F][d], [F]
    const void* w_2;   const float* b_2;     // [d][F], [d]
    const float* ln2_g; const float* ln2_b;  // [d]
};

struct HeadW {  // all fp32 (exact copies of the blob values)
    const float *E, *v_w, *b_w, *v_mu, *b_mu, *v_s, *b_s, *v_k1, *b_k1, *v_k2, *b_k2;
};

// The same model with every matrix transposed to [in][out] (storage type for
// the layer matrices, fp32 for the head) so that a warp whose lanes own
// consecutive outputs reads consecutive words.  Self-contained: all vectors
// are copied in too, and every pointer lies in [base, base + bytes).
struct DevModelT {
    const float* type_emb;   // [K][d]
    const double* tenc;      // [2d] temporal encoding: phases a_j, then frequencies b_j
    LayerW layer[MAX_LAYERS];  // w_qkv [d][3d], w_o [d][d], w_1 [d][F], w_2 [F][d]
    HeadW head;              // E [d][3d], v_w/v_mu/v_s [d][M], v_k1 [d][d], v_k2 [d][K]
    const char* base;
    size_t bytes;
    // lane-packed copy only (null in the transposed one):
    const float* tenc_ff;    // [4][d] fp32 pairs of the encoding table: a_hi, a_lo, b_hi, b_lo
    const float* head_t;     // [3M][d] lane-packed [V_w E_1; V_mu E_2; V_s E_3] (products in fp64)
    const float* head_tb;    // [3M] b_w, b_mu, b_s
};

// One model on the device.  Every pointer lies in [base, base + bytes), so a
// kernel can copy the whole model to shared memory and rebase the pointers.
struct DevModel {
    int L, d, nh, dh, F, M, K, dtype;
    int enc;                 // encoder: 0 THP, 1 SAHP, 2 AttNHP (App. D.4)
    int v_f16;               // V cache stored as fp16 (the bf16-rounded values, for the
                             // fp16 x fp16 second product of the tcgen05 attention)
    int attn_tc;             // attention on the tcgen05 kernel (else the mma.sync one)
    int tenc_paired;         // dims 2i and 2i+1 share one angle (THP, AttNHP)
    const float* type_emb;   // [K][d] fp32
    // temporal encoding z_j = sin / cos (a_j + b_j t) for even / odd j:
    // [2d] phases a_j then frequencies b_j (fp64)
    const double* tenc;
    LayerW layer[MAX_LAYERS];
    HeadW head;
    const char* base;
    size_t bytes;
    const float* head_ek_w;  // [4d][d] fp32: rows of E then rows of v_k1
    const float* head_ek_b;  // [4d]: zeros then b_k1
    const float* head_out_t; // [d][3M+K] fp32: v_w, v_mu, v_s, v_k2 transposed side by side
    const float* head_out_b; // [3M+K]: b_w, b_mu, b_s, b_k2
    const float* head_out_g; // the same maps group by group: [d][M] x 3, then [d][K] (contiguous)
    const void* head_ek_hi;  // [4d][d] bf16: head_ek_w = hi + lo (split of each fp32 value)
    const void* head_ek_lo;
    DevModelT t;             // transposed copy (read by the per-sequence draft kernel)
    // Lane-packed copy (same struct, read by the lane form of the draft
    // kernel): a matrix W [out][in] is stored as chunks of CH = 16 / sizeof
    // (element) consecutive inputs, chunk c of output j at element
    // (c * out + j) * CH, so the lanes of a warp that own consecutive outputs
    // read consecutive 16-byte words.  Vectors as in the other copies.
    DevModelT p;
    __host__ __device__ int head_width() const { return 3 * M + K; }
};

// KV cache of one model: K and V each [L][Bmax][nh][n_max][dh] (storage type).
struct KVCache {
    void* k;
    void* v;
    int Bmax, n_max;
};

// Parameters of one sampling call, kept in device memory so that one
// captured graph serves every call with the same (batch, gamma, flags).
struct CallParams {
    int B, H, N, gamma, n_max;
    uint32_t flags;
    uint64_t seed;
    float* out_tau;
    double* out_t;
    int* out_k;
    int max_loops;
    // End-time stop rule (Alg. 1): with out_count set, a sequence stops once
    // its last event lies beyond t_end (or after N events); only events with
    // t <= t_end are written and out_count[s] receives their number.
    double t_end;
    int* out_count;
    // Poisson draft (App. D.3): rate, its log, and log p of the marks [K]
    float pois_rate, pois_log_rate;
    const float* pois_logp;
    // iteration cap of the Theorem-1 resampling loop (65 536 unless lowered
    // by tppsd_set_limits)
    int resample_cap;
    // TPPSD_FLAG_DEBUG_TRACE: [Bmax][n_max] records of the verify decisions
    // at each absolute position (null when off)
    float4* trace;
};

// Device counters of the current call (mirrors tppsd_stats + status).
struct DevStats {
    unsigned long long rounds, drafted, accepted, emitted, resample_iters, cap_hits, loop_iters;
    unsigned long long target_keys;  // sum over (sequence, target pass) of keys per layer
    unsigned long long draft_keys;   // sum over draft encode steps of keys per layer
    int round_limit_hit;
};

// Kernel classes timed by the profiling loop.
enum KernelClass {
    KC_DRAFT = 0, KC_EMBED, KC_GEMM_QKV, KC_ATTENTION, KC_GEMM_O, KC_LAYERNORM, KC_GEMM_FFN1,
    KC_GEMM_FFN2, KC_HEAD, KC_EPILOGUE, KC_AR_SAMPLE, KC_CONTROL, KC_BEGIN, KC_COUNT
};

// Optional launch timer: mark(cls, 1) before a launch, mark(cls, 0) after.
struct Prof {
    void (*mark)(void* self, int cls, int begin, cudaStream_t st);
    void* self;
};
#define PROF_MARK(prof, cls, b, st) \
    do {                            \
        if (prof) (prof)->mark((prof)->self, (cls), (b), (st)); \
    } while (0)

// Per-sequence state of the sampler.
struct SeqState {
    float* tau;   // [Bmax][n_max] inter-event times
    double* t;    // [Bmax][n_max] absolute times
    int* k;       // [Bmax][n_max] marks
    int* n_emit;  // [Bmax] events so far (history + generated)
    int* n_draft; // [Bmax] positions encoded in the draft cache
    int* done;    // [Bmax]
    int n_max;
};

// Device memory of the split-key form: partial results and arrival counters
// (zeroed once; every launch leaves them zero).  Null: no splits.
struct AttnScratch {
    float* part;
    size_t part_bytes;
    int* cnt;
    long long cnt_items;
};

// Row workspace of the batched forward.
struct Work {
    int* err;            // device error flag for bounded waits (may be null)
    int R;               // capacity in rows
    int* row_seq;        // [R] sequence of the row, -1 = inactive
    int* row_pos;        // [R] absolute position of the row
    float* x;            // [R][dmax] residual stream (fp32)
    void* xb;            // [R][dmax] GEMM input copy (storage type)
    void* q;             // [R][dmax]
    void* att;           // [R][dmax]
    void* hid;           // [R][Fmax]
    float* y;            // [R][dmax] pre-LayerNorm sums
    float* heads;        // [R][hw_max]
    float* hd4;          // [R][4 dmax] head pre-activations (e = E h, V_k1 h + b_k1)
    AttnScratch attn;    // split-key attention scratch (may be empty)
};

// Row modes of a forward pass.
enum RowMode { ROWS_STEP = 0, ROWS_SPAN = 1 };
struct RowSpec {
    int mode;   // ROWS_STEP: r = s*q + l at position n_emit[s]-1+l (skips done s)
                // ROWS_SPAN: g = g0 + r, s = g / q, position g % q
    int q;      // rows per sequence
    int count;  // rows in this pass
    int g0;
    int pre_embedded;  // ROWS_STEP: the rows (x, xb, row_seq, row_pos) were written by the draft kernel
};

// Arguments of one attention launch (rows of q_per_seq queries per sequence).
template <typename T>
struct AttArgs {
    const T* q;   // [R][d]
    const T* kc;  // K cache base ([layer][seq][head][pos][d_head])
    const T* vc;
    T* out;       // [R][d]
    const int* row_seq;
    const int* row_pos;
    int count, q_per_seq, g0, d, nh, layer;
    KVCache kv;
    float scale;
    // AttNHP (App. D.4): normaliser 1 + sum f, and instead of `out` the
    // residual h <- h + tanh(a) into x (fp32 [R][d]) and its rounded copy
    // into the h half of the [z | h] rows hb ([R][2d])
    int attnhp;
    float* x;
    T* hb;
};
// KV cache [items * n_max rows][dh] (bf16, or fp16 with f16) as a 2-D
// tensor map with boxes of box_rows rows, swizzled by the row width.
bool kv_tile_map(CUtensorMap* m, const void* base, int dh, int n_max, long long items, int box_rows, int f16 = 0);
cudaError_t launch_attn_mma(const AttArgs<__nv_bfloat16>& a, int dh, int nh, int nseg, int* err,
                            cudaStream_t st);

// Attention on the tcgen05 tensor cores (attn_tc.cu).  Device arguments of
// one launch; the K / V / Q tensor maps are passed beside them.
struct AttTcArgs {
    const int* row_seq;
    const int* row_pos;
    __nv_bfloat16* out;   // [R][d] attention output (softmax layers)
    float* x;             // AttNHP: residual h (fp32 [R][d]) ...
    __nv_bfloat16* hb;    // ... and its rounded copy in the [z | h] rows ([R][2d])
    int count, q_per_seq, g0, d, nh, layer, Bmax, n_max, attnhp;
    float c2;             // 1/sqrt(d_head) * log2(e): scores in base-2 units
    float slack;          // a tile whose scores exceed the reference by more starts a new one
    int nsplit;           // key splits per item (flash-decoding)
    float* part;          // [items * nsplit][NQ * (d_head + 2)] partial results
    int* cnt;             // [items] arrival counters, zero between launches
    int* err;
};
int attn_tc_supported(int dh);
// Key splits per item of a step pass of `items` (query block, head,
// sequence) items over a cache of n_max positions.
long long attn_splits(long long items, int n_max, int dh, int nq, int n_sm);
// step_rows: one pass of gamma+1 (or 1) rows per sequence, where key splits
// are allowed; prefill and scoring passes use one CTA per query block.
cudaError_t launch_attn_tc(const AttArgs<__nv_bfloat16>& a, int dh, int nh, int nseg, bool step_rows,
                           const AttnScratch& sc, int* err, cudaStream_t st);

// ---------------------------------------------------------------- tensor-core GEMM
enum { EPI_TC_QKV = 0, EPI_TC_RELU = 1, EPI_TC_RESID_LN = 2, EPI_TC_F32 = 3 };
struct TcGemmArgs {
    int R, N, K, epi;
    const float* bias;
    // EPI_TC_QKV
    __nv_bfloat16* q_out; __nv_bfloat16* kc; __nv_bfloat16* vc;
    const int* row_seq; const int* row_pos;
    int d, nh, dh, layer, Bmax, n_max;
    // EPI_TC_RELU
    __nv_bfloat16* out_t;
    // EPI_TC_RESID_LN
    const float* resid; float* x_out; __nv_bfloat16* xb_out; const float* ln_g; const float* ln_b;
    int* err;  // set (first error wins) if a pipeline wait times out
    int stall; // diagnostic: wait on a barrier nothing completes, so the bounded wait runs out
    int v_f16; // EPI_TC_QKV: V stored as fp16 (of the bf16-rounded value)
    // EPI_TC_F32: fp32 out [R][N] = acc + b
    float* out_f;
    // split: fp32-accurate product of fp32 operands given as bf16 pairs, as
    // one GEMM over K' = 3K: [A_hi | A_hi | A_lo] [W_hi | W_lo | W_hi]^T
    // (second maps: A_lo, W_lo)
    int split;
};
struct TcLayerMaps {
    CUtensorMap wqkv, wo, w1, w2;      // boxes of the separate GEMMs
    CUtensorMap wo_m, w1_m, w2_m;      // boxes of 128 rows for the fused block
    CUtensorMap wqkv_f;                // W_qkv with boxes of mlp_cl_qkv_cols rows (folded QKV)
};
// Tensor maps of one bf16 model's weights and of the row-workspace buffers it
// reads (rows = Work.R), built once per context.
struct TcPlan {
    int enabled;
    int bn_qkv, bn_o, bn_ffn1;  // bn_o: columns per CTA of the cluster LayerNorm GEMMs
    int mlp;                    // post-attention block by the fused kernel
    int mlp_cl;                 // ... in its cluster form (FFN split over F / 128 CTAs)
    int qkv_fold;               // ... which also computes the next layer's Q, K, V
    int head;                   // heads by the tensor-core head kernel (d = 128)
    CUtensorMap head_hi, head_lo;
    // other widths: [E; V_k1] h by the split GEMM (A_hi = xb, A_lo = att), then
    // the small maps by k_head_out
    int head_g, bn_head;
    CUtensorMap head_hi_g, head_lo_g;
    int* err;
    int stall;                  // diagnostic stall of the QKV GEMM (TcGemmArgs.stall)
    CUtensorMap a_xb, a_att, a_hid;
    CUtensorMap a_zh;           // [R][2d] view of the [z | h] rows (AttNHP QKV input)
    TcLayerMaps layer[MAX_LAYERS];
};
bool make_tmap_bf16(CUtensorMap* map, const void* ptr, int K, int rows, int box_rows);
// The driver's cuTensorMapEncodeTiled (null if unavailable).
PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder();
cudaError_t launch_gemm_tc(const CUtensorMap& A, const CUtensorMap& W, const TcGemmArgs& a, int BN,
                           cudaStream_t st);
// The split form (a.split = 1): A2 = A_lo, W2 = W_lo.
cudaError_t launch_gemm_tc_split(const CUtensorMap& A, const CUtensorMap& A2, const CUtensorMap& W,
                                 const CUtensorMap& W2, const TcGemmArgs& a, int BN, cudaStream_t st);
// Fused post-attention block of a layer (mlp_tc.cu): x1 = LN1(x + att W_o^T
// + b_o); x = LN2(x1 + relu(x1 W_1^T + b_1) W_2^T + b_2); xb = bf16(x).
struct MlpArgs {
    int R, F;
    const float *b_o, *ln1_g, *ln1_b, *b_1, *b_2, *ln2_g, *ln2_b;
    float* x;             // [R][d] residual in, LN2 output out
    __nv_bfloat16* xb;    // [R][d] bf16 copy of the output
    int* err;
    // qkv (cluster form): also the next layer's Q, K, V from the output rows,
    // stored as the QKV GEMM's epilogue stores them
    int qkv;
    const float* b_qkv;   // [3d] the next layer's bias
    __nv_bfloat16* q_out; __nv_bfloat16* kc; __nv_bfloat16* vc;
    const int* row_seq; const int* row_pos;
    int nh, dh, layer, Bmax, n_max, v_f16;
};
int mlp_tc_supported(int d, int F);
int mlp_cl_supported(int d, int F);
// Columns of W_qkv per CTA when the cluster form can fold the next layer's
// QKV GEMM in (0: it cannot); the W_qkv tensor map then has boxes of that
// many rows.
int mlp_cl_qkv_cols(int d, int F);
cudaError_t launch_mlp_cl(const CUtensorMap& att, const CUtensorMap& wo, const CUtensorMap& w1,
                          const CUtensorMap& w2, const CUtensorMap& wq, const MlpArgs& a, cudaStream_t st);
// att: tensor map of the attention output rows (box 64 x 128); wo / w1 / w2:
// weight maps with boxes of 64 x 128.
cudaError_t launch_mlp_tc(const CUtensorMap& att, const CUtensorMap& wo, const CUtensorMap& w1,
                          const CUtensorMap& w2, const MlpArgs& a, cudaStream_t st);
// Target heads on the tensor cores (head_tc.cu) for bf16 models with d = 128:
// reads the final hidden rows w.x, writes w.heads for rows with row_seq >= 0.
// hi / lo: tensor maps of the split [E; V_k1] (boxes of 64 x 128).
int head_tc_supported(const DevModel& m);
cudaError_t launch_head_tc(const CUtensorMap& hi, const CUtensorMap& lo, const DevModel& m, const Work& w, int R,
                           cudaStream_t st);
// Columns per CTA of the cluster LayerNorm GEMM for a row width N (0: unsupported).
int ln_cluster_cols(int N);
// EPI_TC_RESID_LN by a cluster of N / ln_cluster_cols(N) CTAs per 128 rows;
// W's tensor map has boxes of ln_cluster_cols(N) rows.
cudaError_t launch_gemm_ln_cluster(const CUtensorMap& A, const CUtensorMap& W, const TcGemmArgs& a,
                                   cudaStream_t st);

// ---------------------------------------------------------------- launchers
// All return cudaGetLastError() of their launches.
cudaError_t launch_forward(const DevModel& m, const KVCache& kv, const SeqState& ss,
                           const Work& w, const RowSpec& rs, bool want_heads,
                           cudaStream_t st, int* launches, const Prof* prof,
                           const TcPlan* tc = nullptr);
cudaError_t launch_history_times(const SeqState& ss, int B, int H, cudaStream_t st);
cudaError_t launch_begin(const CallParams& p, CallParams* dp, const SeqState& ss,
                         DevStats* stats, cudaStream_t st);
cudaError_t launch_draft(const DevModel& m, const KVCache& kv, const SeqState& ss,
                         const CallParams* dp, int B, int gamma, float* draft_heads,
                         int gamma_max, DevStats* stats, cudaStream_t st);
cudaError_t launch_verify_epilogue(const DevModel& mT, const DevModel& mD, const SeqState& ss,
                                   const CallParams* dp, int B, int gamma, const float* t_heads,
                                   const float* d_heads, int gamma_max, DevStats* stats,
                                   cudaStream_t st, bool poisson = false);
cudaError_t launch_poisson_draft(const SeqState& ss, const CallParams* dp, int B, int gamma, int K,
                                 cudaStream_t st);
cudaError_t launch_ar_sample(const DevModel& mT, const SeqState& ss, const CallParams* dp,
                             int B, const float* heads, DevStats* stats, cudaStream_t st);
cudaError_t launch_round_control(const SeqState& ss, const CallParams* dp, int B,
                                 DevStats* stats, unsigned long long cond_handle, int use_cond,
                                 int* active_out, cudaStream_t st);
cudaError_t launch_score_survival(const DevModel& m, const SeqState& ss, const Work& w, int B, int len,
                                  int g0, int rows, double t_end, double* out_logS, cudaStream_t st);
cudaError_t launch_score_logs(const DevModel& m, const SeqState& ss, const Work& w, int B,
                              int len, int q, int s0, int rows, float* out_heads, float* out_logg,
                              float* out_logf, cudaStream_t st);
size_t draft_smem_bytes(const DevModel& m, bool stage_weights);
// One-CTA-per-sequence draft (draft.cu) for the shapes it is compiled for.
int draft_team_supported(const DevModel& m);
// Lane form of the draft kernel (draft.cu) for d <= 32 models whose packed
// copy and two sequences' draft KV fit in shared memory.
int draft_lane_supported(const DevModel& m, int n_max, int gamma_max);
// The target's embedding of the verify rows (THP / SAHP layout), written by
// the lane draft kernel in place of the forward's embedding kernel: row
// s (gamma + 1) + l is the event at position n_emit[s] - 1 + l.
struct DraftEmbed {
    const double* tenc;     // the target's encoding table (a_j, then b_j)
    const float* type_emb;  // [K][d]
    float* x;               // [rows][d] fp32
    void* xb;               // [rows][d] storage type (the draft's, equal to the target's)
    int* row_seq;
    int* row_pos;
    int d, K, paired;
};
// emb: null, or the target rows to write (then the forward skips its
// embedding kernel: RowSpec.pre_embedded).
cudaError_t launch_draft_lane(const DevModel& m, const KVCache& kv, const SeqState& ss,
                              const CallParams* dp, int B, int gamma, float* draft_heads,
                              int gamma_max, DevStats* stats, int* err, cudaStream_t st,
                              const DraftEmbed* emb = nullptr);
cudaError_t launch_draft_team(const DevModel& m, const KVCache& kv, const SeqState& ss,
                              const CallParams* dp, int B, int gamma, float* draft_heads,
                              int gamma_max, DevStats* stats, int* err, cudaStream_t st);
int draft_supported(const DevModel& m);

}  // namespace tppsd
