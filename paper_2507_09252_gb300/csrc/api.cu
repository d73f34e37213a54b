// C ABI of the TPP-SD sampler (include/tppsd.h): context, weight upload,
// prefill, the device-resident round loop, scoring, status and stats.
//
// The sampling loop of Alg. 1 runs without host round trips: one round
// (draft -> verify forward -> heads -> epilogue -> control) is captured once
// into the body of a CUDA-graph WHILE node; k_round_control sets the loop
// condition from the device.  Per-call values (history length, event count,
// seed, output pointers) live in device memory, so one instantiated graph
// serves every call with the same (batch, gamma, flags).
#include <cuda_runtime.h>
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <chrono>
#include <cmath>
#include <map>
#include <mutex>
#include <new>
#include <string>
#include <thread>
#include <tuple>
#include <vector>

#include "../../include/tppsd.h"
#include "engine.h"

using namespace tppsd;

namespace {

struct HostModel {
    tppsd_model_cfg cfg{};
    DevModel dm{};
    void* dbuf = nullptr;
    void* tbuf = nullptr;
    void* pbuf = nullptr;
};

struct GraphEntry {
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    int launches_per_round = 0;
};

// CUDA events around every launch of a profiled call, accumulated per class.
struct Profiler {
    std::vector<cudaEvent_t> pool;
    std::vector<std::pair<int, int>> spans;  // (class, index of begin event)
    size_t used = 0;
    int open_cls = -1, open_ev = -1;
    cudaError_t err = cudaSuccess;
    cudaEvent_t next() {
        if (used == pool.size()) {
            cudaEvent_t e;
            cudaError_t r = cudaEventCreate(&e);
            if (r != cudaSuccess) { err = r; return nullptr; }
            pool.push_back(e);
        }
        return pool[used++];
    }
    void reset() { used = 0; spans.clear(); err = cudaSuccess; }
    static void mark(void* self, int cls, int begin, cudaStream_t st) {
        Profiler* p = (Profiler*)self;
        cudaEvent_t e = p->next();
        if (!e) return;
        cudaError_t r = cudaEventRecord(e, st);
        if (r != cudaSuccess) p->err = r;
        if (begin) p->spans.emplace_back(cls, (int)(p->used - 1));
    }
};

// Iteration cap of the Theorem-1 resampling loop: the paper's loop is
// unbounded; the cap keeps the kernel's run time bounded (the bias it can
// introduce is at most the probability of (1 - TV)^cap).
constexpr int DEFAULT_RESAMPLE_CAP = 65536;

}  // namespace

struct tppsd_ctx {
    int device = 0;
    HostModel T, D;
    int max_batch = 0, n_max = 0, max_gamma = 0;
    SeqState ss{};
    KVCache kvT{}, kvD{};
    Work work{};
    float* draft_heads = nullptr;
    CallParams* d_params = nullptr;
    float* d_pois_logp = nullptr;  // [MAX_MARKS] log p of the Poisson draft
    DevStats* d_stats = nullptr;
    int* d_active = nullptr;
    int* h_active = nullptr;  // pinned
    cudaStream_t cap_stream = nullptr;
    cudaEvent_t done_event = nullptr;
    cudaStream_t last_stream = nullptr;
    std::map<std::tuple<int, int, int, unsigned>, GraphEntry> graphs;
    // staging of host outputs
    void* stage = nullptr;
    size_t stage_bytes = 0;
    // state
    int prefill_batch = 0, hist_len = 0;
    bool prefilled = false;
    int last_launches = 0;
    int prefill_launches = 0;
    Profiler prof;
    bool profiled = false;
    TcPlan tc{};          // tensor-core GEMM plan of the target model (enabled if supported)
    int* d_err = nullptr; // device error code of the current call (pipeline wait timeouts)
    int resample_cap = DEFAULT_RESAMPLE_CAP;  // Theorem-1 loop cap (tppsd_set_limits)
    float4* d_trace = nullptr;  // [max_batch][n_max] decision records (TPPSD_FLAG_DEBUG_TRACE)
    int trace_batch = 0, trace_hist = 0, trace_events = 0;  // extent of the last traced call
    int max_rounds = 0;   // round-loop cap below the natural N + 2 (0: none)
    std::string err;
    std::vector<void*> allocs;
};

// ---------------------------------------------------------------- helpers
namespace tppsd {
int g_pdl = 1;
}  // namespace tppsd

static const char* fault_mode() {
    const char* f = getenv("TPPSD_FAULT");
    return f ? f : "";
}

#define CK(expr)                                                                   \
    do {                                                                           \
        cudaError_t e_ = (expr);                                                   \
        if (e_ != cudaSuccess) {                                                   \
            if (ctx) ctx->err = std::string(#expr) + ": " + cudaGetErrorString(e_); \
            return e_ == cudaErrorMemoryAllocation ? TPPSD_ERR_OOM : TPPSD_ERR_CUDA; \
        }                                                                          \
    } while (0)

static bool is_device_ptr(const void* p) {
    if (!p) return false;
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

static bool cfg_ok(const tppsd_model_cfg* c) {
    if (!c) return false;
    if (c->layers < 1 || c->layers > MAX_LAYERS) return false;
    if (c->d_model < 16 || c->d_model > MAX_D || c->d_model % 16) return false;
    if (c->heads < 1 || c->heads > 8 || c->d_model % c->heads) return false;
    const int dh = c->d_model / c->heads;
    if (dh != 8 && dh != 16 && dh != 32 && dh != 64) return false;
    if (c->d_ffn < 16 || c->d_ffn > 4096 || c->d_ffn % 16) return false;
    if (c->n_mix < 1 || c->n_mix > MAX_MIX) return false;
    if (c->n_marks < 1 || c->n_marks > MAX_MARKS) return false;
    if (c->encoder < 0 || c->encoder > 2) return false;
    return c->dtype == 0 || c->dtype == 1;
}

extern "C" size_t tppsd_blob_floats(const tppsd_model_cfg* c) {
    if (!cfg_ok(c)) return 0;
    const size_t L = c->layers, d = c->d_model, F = c->d_ffn, M = c->n_mix, K = c->n_marks;
    const size_t layer = c->encoder == 2 ? 3 * d * 2 * d + 3 * d
                                         : 3 * d * d + 3 * d + d * d + d + 2 * d + F * d + F + d * F + d + 2 * d;
    const size_t tail = c->encoder == 1 ? d : c->encoder == 2 ? 2 : 0;
    return K * d + L * layer + 3 * d * d + 3 * (M * d + M) + d * d + d + K * d + K + tail;
}

static uint16_t f32_to_bf16_bits(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    u += 0x7FFFu + ((u >> 16) & 1u);  // nearest, ties to even (finite inputs)
    return (uint16_t)(u >> 16);
}

// Lays one model out in a single device buffer: storage-type GEMM matrices
// first, then fp32 vectors, embeddings and head, then the fp64 frequency
// table; every piece 16-byte aligned.
static tppsd_status_t upload_model(tppsd_ctx* ctx, HostModel& hm, const tppsd_model_cfg* cfg,
                                   const float* blob_any, size_t nfloats) {
    hm.cfg = *cfg;
    const int L = cfg->layers, d = cfg->d_model, F = cfg->d_ffn, M = cfg->n_mix, K = cfg->n_marks;
    const int enc = cfg->encoder;
    const bool att = enc == 2;             // AttNHP: QKV over [z; h] only
    const size_t din = att ? 2 * (size_t)d : (size_t)d;
    std::vector<float> blob(nfloats);
    if (is_device_ptr(blob_any)) {
        CK(cudaMemcpy(blob.data(), blob_any, nfloats * sizeof(float), cudaMemcpyDeviceToHost));
    } else {
        memcpy(blob.data(), blob_any, nfloats * sizeof(float));
    }
    // blob offsets (include/tppsd.h layout)
    size_t o = 0;
    auto take = [&](size_t n) { size_t r = o; o += n; return r; };
    const size_t o_emb = take((size_t)K * d);
    struct LO { size_t wqkv, bqkv, wo, bo, g1, b1n, w1, b1, w2, b2, g2, b2n; };
    std::vector<LO> lo(L);
    for (int l = 0; l < L; ++l) {
        lo[l].wqkv = take(3 * (size_t)d * din); lo[l].bqkv = take(3 * d);
        if (att) continue;
        lo[l].wo = take((size_t)d * d); lo[l].bo = take(d);
        lo[l].g1 = take(d); lo[l].b1n = take(d);
        lo[l].w1 = take((size_t)F * d); lo[l].b1 = take(F);
        lo[l].w2 = take((size_t)d * F); lo[l].b2 = take(d);
        lo[l].g2 = take(d); lo[l].b2n = take(d);
    }
    const size_t oE = take(3 * (size_t)d * d);
    const size_t ovw = take((size_t)M * d), obw = take(M), ovm = take((size_t)M * d), obm = take(M);
    const size_t ovs = take((size_t)M * d), obs = take(M);
    const size_t ok1 = take((size_t)d * d), obk1 = take(d), ok2 = take((size_t)K * d), obk2 = take(K);
    const size_t o_tail = take(enc == 1 ? d : att ? 2 : 0);
    if (o != nfloats) {
        ctx->err = "blob size does not match the model shape";
        return TPPSD_ERR_INVALID_ARG;
    }
    std::vector<char> buf;
    auto add = [&](const void* src, size_t bytes) {
        size_t off = (buf.size() + 15) & ~(size_t)15;
        buf.resize(off + bytes);
        memcpy(buf.data() + off, src, bytes);
        return off;
    };
    const bool bf = cfg->dtype == 1;
    auto add_mat = [&](size_t off, size_t n) {
        if (!bf) return add(blob.data() + off, n * sizeof(float));
        std::vector<uint16_t> t(n);
        for (size_t i = 0; i < n; ++i) t[i] = f32_to_bf16_bits(blob[off + i]);
        return add(t.data(), n * 2);
    };
    auto add_vec = [&](size_t off, size_t n) { return add(blob.data() + off, n * sizeof(float)); };
    struct LB { size_t wqkv, bqkv, wo, bo, g1, b1n, w1, b1, w2, b2, g2, b2n; };
    std::vector<LB> lb(L);
    for (int l = 0; l < L; ++l) {
        lb[l].wqkv = add_mat(lo[l].wqkv, 3 * (size_t)d * din);
        if (att) continue;
        lb[l].wo = add_mat(lo[l].wo, (size_t)d * d);
        lb[l].w1 = add_mat(lo[l].w1, (size_t)F * d);
        lb[l].w2 = add_mat(lo[l].w2, (size_t)d * F);
    }
    for (int l = 0; l < L; ++l) {
        lb[l].bqkv = add_vec(lo[l].bqkv, 3 * d);
        if (att) continue;
        lb[l].bo = add_vec(lo[l].bo, d);
        lb[l].g1 = add_vec(lo[l].g1, d); lb[l].b1n = add_vec(lo[l].b1n, d);
        lb[l].b1 = add_vec(lo[l].b1, F); lb[l].b2 = add_vec(lo[l].b2, d);
        lb[l].g2 = add_vec(lo[l].g2, d); lb[l].b2n = add_vec(lo[l].b2n, d);
    }
    const size_t b_emb = add_vec(o_emb, (size_t)K * d);
    const size_t bE = add_vec(oE, 3 * (size_t)d * d);
    const size_t bvw = add_vec(ovw, (size_t)M * d), bbw = add_vec(obw, M);
    const size_t bvm = add_vec(ovm, (size_t)M * d), bbm = add_vec(obm, M);
    const size_t bvs = add_vec(ovs, (size_t)M * d), bbs = add_vec(obs, M);
    const size_t bk1 = add_vec(ok1, (size_t)d * d), bbk1 = add_vec(obk1, d);
    const size_t bk2 = add_vec(ok2, (size_t)K * d), bbk2 = add_vec(obk2, K);
    // temporal encoding (App. D.4): z_j = sin / cos (a_j + b_j t), je = j - j mod 2
    std::vector<double> tenc(2 * (size_t)d, 0.0);
    if (att && !(blob[o_tail] > 0.f && blob[o_tail + 1] > 0.f)) {
        ctx->err = "AttNHP time scales must be positive";
        return TPPSD_ERR_INVALID_ARG;
    }
    for (int j = 0; j < d; ++j) {
        const double je = (double)(j - (j & 1)), e = je / (double)d;
        if (enc == 1) {          // SAHP: phase j / 10000^(je/d), learned frequency w_j
            tenc[j] = (double)j / pow(10000.0, e);
            tenc[d + j] = (double)blob[o_tail + j];
        } else if (att) {        // AttNHP: wavelength m (5M/m)^(je/d)
            const double sm = blob[o_tail], sM = blob[o_tail + 1];
            tenc[d + j] = 1.0 / (sm * pow(5.0 * sM / sm, e));
        } else {                 // THP: frequency 10000^(-je/d)
            tenc[d + j] = pow(10000.0, -e);
        }
    }
    const size_t b_om = add(tenc.data(), tenc.size() * sizeof(double));
    // head matrices regrouped for the batched head: [E; v_k1] (4d x d) with
    // bias [0; b_k1], and the output maps transposed side by side (d x (3M+K))
    std::vector<float> ek((size_t)4 * d * d), ekb((size_t)4 * d, 0.f);
    memcpy(ek.data(), blob.data() + oE, sizeof(float) * 3 * (size_t)d * d);
    memcpy(ek.data() + 3 * (size_t)d * d, blob.data() + ok1, sizeof(float) * (size_t)d * d);
    memcpy(ekb.data() + 3 * d, blob.data() + obk1, sizeof(float) * d);
    const int WO = 3 * M + K;
    std::vector<float> ho((size_t)d * WO), hob(WO);
    const size_t src_off[4] = {ovw, ovm, ovs, ok2}, bsrc[4] = {obw, obm, obs, obk2};
    const int cnt[4] = {M, M, M, K};
    for (int part = 0, col0 = 0; part < 4; col0 += cnt[part], ++part)
        for (int o2 = 0; o2 < cnt[part]; ++o2) {
            hob[col0 + o2] = blob[bsrc[part] + o2];
            for (int i = 0; i < d; ++i) ho[(size_t)i * WO + col0 + o2] = blob[src_off[part] + (size_t)o2 * d + i];
        }
    const size_t b_ek = add(ek.data(), ek.size() * 4), b_ekb = add(ekb.data(), ekb.size() * 4);
    const size_t b_ho = add(ho.data(), ho.size() * 4), b_hob = add(hob.data(), hob.size() * 4);
    std::vector<float> hog((size_t)d * WO);  // group by group, [d][cnt] each
    for (int part = 0, col0 = 0; part < 4; col0 += cnt[part], ++part)
        for (int i = 0; i < d; ++i)
            for (int o2 = 0; o2 < cnt[part]; ++o2)
                hog[(size_t)d * col0 + (size_t)i * cnt[part] + o2] = ho[(size_t)i * WO + col0 + o2];
    const size_t b_hog = add(hog.data(), hog.size() * 4);
    // [E; v_k1] as a sum of two bf16 matrices (hi + lo) for the tensor-core head
    std::vector<uint16_t> ekh(ek.size()), ekl(ek.size());
    for (size_t i = 0; i < ek.size(); ++i) {
        ekh[i] = f32_to_bf16_bits(ek[i]);
        uint32_t hb = (uint32_t)ekh[i] << 16;
        float hf;
        memcpy(&hf, &hb, 4);
        ekl[i] = f32_to_bf16_bits(ek[i] - hf);
    }
    const size_t b_ekh = add(ekh.data(), ekh.size() * 2), b_ekl = add(ekl.data(), ekl.size() * 2);
    buf.resize((buf.size() + 15) & ~(size_t)15);
    CK(cudaMalloc(&hm.dbuf, buf.size()));
    ctx->allocs.push_back(hm.dbuf);
    CK(cudaMemcpy(hm.dbuf, buf.data(), buf.size(), cudaMemcpyHostToDevice));
    const char* b = (const char*)hm.dbuf;
    DevModel& m = hm.dm;
    m.L = L; m.d = d; m.nh = cfg->heads; m.dh = d / cfg->heads; m.F = F; m.M = M; m.K = K;
    m.dtype = cfg->dtype;
    m.enc = enc;
    m.tenc_paired = enc != 1;
    m.type_emb = (const float*)(b + b_emb);
    m.tenc = (const double*)(b + b_om);
    for (int l = 0; l < L; ++l) {
        LayerW& w = m.layer[l];
        w = LayerW{};
        w.w_qkv = b + lb[l].wqkv; w.b_qkv = (const float*)(b + lb[l].bqkv);
        if (att) continue;
        w.w_o = b + lb[l].wo; w.b_o = (const float*)(b + lb[l].bo);
        w.ln1_g = (const float*)(b + lb[l].g1); w.ln1_b = (const float*)(b + lb[l].b1n);
        w.w_1 = b + lb[l].w1; w.b_1 = (const float*)(b + lb[l].b1);
        w.w_2 = b + lb[l].w2; w.b_2 = (const float*)(b + lb[l].b2);
        w.ln2_g = (const float*)(b + lb[l].g2); w.ln2_b = (const float*)(b + lb[l].b2n);
    }
    HeadW& h = m.head;
    h.E = (const float*)(b + bE);
    h.v_w = (const float*)(b + bvw); h.b_w = (const float*)(b + bbw);
    h.v_mu = (const float*)(b + bvm); h.b_mu = (const float*)(b + bbm);
    h.v_s = (const float*)(b + bvs); h.b_s = (const float*)(b + bbs);
    h.v_k1 = (const float*)(b + bk1); h.b_k1 = (const float*)(b + bbk1);
    h.v_k2 = (const float*)(b + bk2); h.b_k2 = (const float*)(b + bbk2);
    m.head_ek_w = (const float*)(b + b_ek);
    m.head_ek_b = (const float*)(b + b_ekb);
    m.head_out_t = (const float*)(b + b_ho);
    m.head_out_b = (const float*)(b + b_hob);
    m.head_out_g = (const float*)(b + b_hog);
    m.head_ek_hi = (const void*)(b + b_ekh);
    m.head_ek_lo = (const void*)(b + b_ekl);
    m.base = b;
    m.bytes = buf.size();
    // transposed, self-contained copy ([in][out] matrices)
    std::vector<char> tb;
    auto tadd = [&](const void* src, size_t bytes) {
        size_t off = (tb.size() + 15) & ~(size_t)15;
        tb.resize(off + bytes);
        memcpy(tb.data() + off, src, bytes);
        return off;
    };
    auto tmat = [&](size_t off, size_t rows, size_t cols, bool storage) {  // blob [rows][cols] -> [cols][rows]
        if (storage && bf) {
            std::vector<uint16_t> t(rows * cols);
            for (size_t r = 0; r < rows; ++r)
                for (size_t c2 = 0; c2 < cols; ++c2) t[c2 * rows + r] = f32_to_bf16_bits(blob[off + r * cols + c2]);
            return tadd(t.data(), t.size() * 2);
        }
        std::vector<float> t(rows * cols);
        for (size_t r = 0; r < rows; ++r)
            for (size_t c2 = 0; c2 < cols; ++c2) t[c2 * rows + r] = blob[off + r * cols + c2];
        return tadd(t.data(), t.size() * 4);
    };
    auto tvec = [&](size_t off, size_t n) { return tadd(blob.data() + off, n * sizeof(float)); };
    std::vector<LB> tl(L);
    for (int l = 0; l < L; ++l) {
        tl[l].wqkv = tmat(lo[l].wqkv, 3 * (size_t)d, din, true);
        if (att) continue;
        tl[l].wo = tmat(lo[l].wo, d, d, true);
        tl[l].w1 = tmat(lo[l].w1, F, d, true);
        tl[l].w2 = tmat(lo[l].w2, d, F, true);
    }
    for (int l = 0; l < L; ++l) {
        tl[l].bqkv = tvec(lo[l].bqkv, 3 * d);
        if (att) continue;
        tl[l].bo = tvec(lo[l].bo, d);
        tl[l].g1 = tvec(lo[l].g1, d); tl[l].b1n = tvec(lo[l].b1n, d);
        tl[l].b1 = tvec(lo[l].b1, F); tl[l].b2 = tvec(lo[l].b2, d);
        tl[l].g2 = tvec(lo[l].g2, d); tl[l].b2n = tvec(lo[l].b2n, d);
    }
    const size_t t_emb = tvec(o_emb, (size_t)K * d);
    const size_t tE = tmat(oE, 3 * (size_t)d, d, false);
    const size_t tvw = tmat(ovw, M, d, false), tbw = tvec(obw, M);
    const size_t tvm = tmat(ovm, M, d, false), tbm = tvec(obm, M);
    const size_t tvs = tmat(ovs, M, d, false), tbs = tvec(obs, M);
    const size_t tk1 = tmat(ok1, d, d, false), tbk1 = tvec(obk1, d);
    const size_t tk2 = tmat(ok2, K, d, false), tbk2 = tvec(obk2, K);
    const size_t t_om = tadd(tenc.data(), tenc.size() * sizeof(double));
    tb.resize((tb.size() + 15) & ~(size_t)15);
    tb.resize((tb.size() + 15) & ~(size_t)15);  // whole 16-byte chunks: one bulk copy stages it
    CK(cudaMalloc(&hm.tbuf, tb.size()));
    ctx->allocs.push_back(hm.tbuf);
    CK(cudaMemcpy(hm.tbuf, tb.data(), tb.size(), cudaMemcpyHostToDevice));
    const char* tbp = (const char*)hm.tbuf;
    DevModelT& mt = m.t;
    mt.type_emb = (const float*)(tbp + t_emb);
    mt.tenc = (const double*)(tbp + t_om);
    for (int l = 0; l < L; ++l) {
        LayerW& w = mt.layer[l];
        w = LayerW{};
        w.w_qkv = tbp + tl[l].wqkv; w.b_qkv = (const float*)(tbp + tl[l].bqkv);
        if (att) continue;
        w.w_o = tbp + tl[l].wo; w.b_o = (const float*)(tbp + tl[l].bo);
        w.ln1_g = (const float*)(tbp + tl[l].g1); w.ln1_b = (const float*)(tbp + tl[l].b1n);
        w.w_1 = tbp + tl[l].w1; w.b_1 = (const float*)(tbp + tl[l].b1);
        w.w_2 = tbp + tl[l].w2; w.b_2 = (const float*)(tbp + tl[l].b2);
        w.ln2_g = (const float*)(tbp + tl[l].g2); w.ln2_b = (const float*)(tbp + tl[l].b2n);
    }
    HeadW& th = mt.head;
    th.E = (const float*)(tbp + tE);
    th.v_w = (const float*)(tbp + tvw); th.b_w = (const float*)(tbp + tbw);
    th.v_mu = (const float*)(tbp + tvm); th.b_mu = (const float*)(tbp + tbm);
    th.v_s = (const float*)(tbp + tvs); th.b_s = (const float*)(tbp + tbs);
    th.v_k1 = (const float*)(tbp + tk1); th.b_k1 = (const float*)(tbp + tbk1);
    th.v_k2 = (const float*)(tbp + tk2); th.b_k2 = (const float*)(tbp + tbk2);
    mt.base = tbp;
    mt.bytes = tb.size();
    // lane-packed, self-contained copy: chunk c (CH consecutive inputs) of
    // output j at element (c * rows + j) * CH, CH = 16 bytes / element
    std::vector<char> pb;
    auto padd = [&](const void* src, size_t bytes) {
        size_t off = (pb.size() + 15) & ~(size_t)15;
        pb.resize(off + bytes);
        memcpy(pb.data() + off, src, bytes);
        return off;
    };
    auto pmat = [&](size_t off, size_t rows, size_t cols, bool storage) {  // blob [rows][cols]
        const bool b16 = storage && bf;
        const size_t CH = b16 ? 8 : 4, nch = (cols + CH - 1) / CH;
        if (b16) {
            std::vector<uint16_t> t(nch * rows * CH, 0);
            for (size_t r = 0; r < rows; ++r)
                for (size_t c2 = 0; c2 < cols; ++c2)
                    t[((c2 / CH) * rows + r) * CH + c2 % CH] = f32_to_bf16_bits(blob[off + r * cols + c2]);
            return padd(t.data(), t.size() * 2);
        }
        std::vector<float> t(nch * rows * CH, 0.f);
        for (size_t r = 0; r < rows; ++r)
            for (size_t c2 = 0; c2 < cols; ++c2) t[((c2 / CH) * rows + r) * CH + c2 % CH] = blob[off + r * cols + c2];
        return padd(t.data(), t.size() * 4);
    };
    auto pvec = [&](size_t off, size_t n) { return padd(blob.data() + off, n * sizeof(float)); };
    std::vector<LB> pl(L);
    for (int l = 0; l < L; ++l) {
        pl[l].wqkv = pmat(lo[l].wqkv, 3 * (size_t)d, din, true);
        if (att) continue;
        pl[l].wo = pmat(lo[l].wo, d, d, true);
        pl[l].w1 = pmat(lo[l].w1, F, d, true);
        pl[l].w2 = pmat(lo[l].w2, d, F, true);
    }
    for (int l = 0; l < L; ++l) {
        pl[l].bqkv = pvec(lo[l].bqkv, 3 * d);
        if (att) continue;
        pl[l].bo = pvec(lo[l].bo, d);
        pl[l].g1 = pvec(lo[l].g1, d); pl[l].b1n = pvec(lo[l].b1n, d);
        pl[l].b1 = pvec(lo[l].b1, F); pl[l].b2 = pvec(lo[l].b2, d);
        pl[l].g2 = pvec(lo[l].g2, d); pl[l].b2n = pvec(lo[l].b2n, d);
    }
    const size_t p_emb = pvec(o_emb, (size_t)K * d);
    const size_t pE = pmat(oE, 3 * (size_t)d, d, false);
    const size_t pvw = pmat(ovw, M, d, false), pbw = pvec(obw, M);
    const size_t pvm = pmat(ovm, M, d, false), pbm = pvec(obm, M);
    const size_t pvs = pmat(ovs, M, d, false), pbs = pvec(obs, M);
    const size_t pk1 = pmat(ok1, d, d, false), pbk1 = pvec(obk1, d);
    const size_t pk2 = pmat(ok2, K, d, false), pbk2 = pvec(obk2, K);
    const size_t p_om = padd(tenc.data(), tenc.size() * sizeof(double));
    // the encoding table as fp32 pairs (hi + lo = the fp64 value to ~48 bits)
    std::vector<float> tff(4 * (size_t)d);
    for (int j = 0; j < d; ++j)
        for (int w = 0; w < 2; ++w) {
            const double v = tenc[(size_t)w * d + j];
            const float hi = (float)v;
            tff[(size_t)(2 * w) * d + j] = hi;
            tff[(size_t)(2 * w + 1) * d + j] = (float)(v - (double)hi);
        }
    const size_t p_tff = padd(tff.data(), tff.size() * 4);
    // time head folded into one map: rows V_w E_1, V_mu E_2, V_s E_3 (fp64
    // products rounded once), bias b_w, b_mu, b_s
    std::vector<float> ht((size_t)3 * M * d), htb((size_t)3 * M);
    const size_t vsrc[3] = {ovw, ovm, ovs}, vb[3] = {obw, obm, obs};
    for (int seg = 0; seg < 3; ++seg)
        for (int j = 0; j < M; ++j) {
            htb[(size_t)seg * M + j] = blob[vb[seg] + j];
            for (int i = 0; i < d; ++i) {
                double acc = 0.0;
                for (int r = 0; r < d; ++r)
                    acc += (double)blob[vsrc[seg] + (size_t)j * d + r] * (double)blob[oE + ((size_t)seg * d + r) * d + i];
                ht[((size_t)seg * M + j) * d + i] = (float)acc;
            }
        }
    std::vector<float> htp(ht.size());
    for (int j = 0; j < 3 * M; ++j)
        for (int i = 0; i < d; ++i) htp[((size_t)(i / 4) * 3 * M + j) * 4 + i % 4] = ht[(size_t)j * d + i];
    const size_t p_ht = padd(htp.data(), htp.size() * 4), p_htb = padd(htb.data(), htb.size() * 4);
    pb.resize((pb.size() + 15) & ~(size_t)15);  // whole 16-byte chunks: one bulk copy stages it
    CK(cudaMalloc(&hm.pbuf, pb.size()));
    ctx->allocs.push_back(hm.pbuf);
    CK(cudaMemcpy(hm.pbuf, pb.data(), pb.size(), cudaMemcpyHostToDevice));
    const char* pbp = (const char*)hm.pbuf;
    DevModelT& mp = m.p;
    mp.type_emb = (const float*)(pbp + p_emb);
    mp.tenc = (const double*)(pbp + p_om);
    for (int l = 0; l < L; ++l) {
        LayerW& w = mp.layer[l];
        w = LayerW{};
        w.w_qkv = pbp + pl[l].wqkv; w.b_qkv = (const float*)(pbp + pl[l].bqkv);
        if (att) continue;
        w.w_o = pbp + pl[l].wo; w.b_o = (const float*)(pbp + pl[l].bo);
        w.ln1_g = (const float*)(pbp + pl[l].g1); w.ln1_b = (const float*)(pbp + pl[l].b1n);
        w.w_1 = pbp + pl[l].w1; w.b_1 = (const float*)(pbp + pl[l].b1);
        w.w_2 = pbp + pl[l].w2; w.b_2 = (const float*)(pbp + pl[l].b2);
        w.ln2_g = (const float*)(pbp + pl[l].g2); w.ln2_b = (const float*)(pbp + pl[l].b2n);
    }
    HeadW& ph = mp.head;
    ph.E = (const float*)(pbp + pE);
    ph.v_w = (const float*)(pbp + pvw); ph.b_w = (const float*)(pbp + pbw);
    ph.v_mu = (const float*)(pbp + pvm); ph.b_mu = (const float*)(pbp + pbm);
    ph.v_s = (const float*)(pbp + pvs); ph.b_s = (const float*)(pbp + pbs);
    ph.v_k1 = (const float*)(pbp + pk1); ph.b_k1 = (const float*)(pbp + pbk1);
    ph.v_k2 = (const float*)(pbp + pk2); ph.b_k2 = (const float*)(pbp + pbk2);
    mp.tenc_ff = (const float*)(pbp + p_tff);
    mp.head_t = (const float*)(pbp + p_ht);
    mp.head_tb = (const float*)(pbp + p_htb);
    mp.base = pbp;
    mp.bytes = pb.size();
    return TPPSD_OK;
}

template <typename P>
static tppsd_status_t dalloc(tppsd_ctx* ctx, P** p, size_t bytes) {
    void* q = nullptr;
    CK(cudaMalloc(&q, bytes ? bytes : 16));
    ctx->allocs.push_back(q);
    *p = (P*)q;
    return TPPSD_OK;
}

#define TRY(x)                               \
    do {                                     \
        tppsd_status_t s_ = (x);             \
        if (s_ != TPPSD_OK) return s_;       \
    } while (0)

static tppsd_status_t alloc_kv(tppsd_ctx* ctx, KVCache& kv, const tppsd_model_cfg& c) {
    const size_t el = c.dtype == 1 ? 2 : 4;
    const size_t n = (size_t)c.layers * ctx->max_batch * ctx->n_max * c.d_model;
    TRY(dalloc(ctx, &kv.k, n * el));
    TRY(dalloc(ctx, &kv.v, n * el));
    // positions never written read as zeros (the attention kernels load whole
    // 128-position tiles and multiply the unused rows by P = 0)
    CK(cudaMemset(kv.k, 0, n * el));
    CK(cudaMemset(kv.v, 0, n * el));
    kv.Bmax = ctx->max_batch;
    kv.n_max = ctx->n_max;
    return TPPSD_OK;
}

// bn for an N-wide GEMM tile: 128 when it gives several tiles, else 256.
static int pick_bn(int N) {
    if (N % 128 == 0 && N <= 512) return 128;
    if (N % 256 == 0) return 256;
    if (N % 128 == 0) return 128;
    if (N % 64 == 0) return 64;
    return 0;
}

// Heads of widths other than 128 (or with the head kernel off): [E; V_k1] h
// by the split tensor-core GEMM over the hi / lo bf16 parts of [E; V_k1].
static void head_gemm_plan(TcPlan& p, const DevModel& m, bool ok, int bn) {
    const int d = m.d;
    p.bn_head = bn;
    const int box = p.bn_head < 256 ? p.bn_head : 256;
    p.head_g = ok && !p.head && p.bn_head && d % 64 == 0 && !getenv("TPPSD_NO_TC_HEAD") &&
               make_tmap_bf16(&p.head_hi_g, m.head_ek_hi, d, 4 * d, box) &&
               make_tmap_bf16(&p.head_lo_g, m.head_ek_lo, d, 4 * d, box);
}

// Tensor maps for the target model's tensor-core GEMMs (bf16 models whose
// widths are multiples of 64 and whose heads are >= 16 wide).
static void build_tc_plan(tppsd_ctx* ctx) {
    TcPlan& p = ctx->tc;
    p.enabled = 0;
    const DevModel& m = ctx->T.dm;
    const tppsd_model_cfg& c = ctx->T.cfg;
    if (getenv("TPPSD_NO_TC") || c.dtype != 1) return;
    const int d = c.d_model, F = c.d_ffn;
    const Work& w = ctx->work;
    if (c.encoder == 2) {  // AttNHP: only the QKV GEMM over the [z | h] rows
        if (d % 64 || m.dh < 16 || !(d == 64 || d == 128 || d == 256 || d == 512)) return;
        p.bn_qkv = d <= 128 ? 64 : pick_bn(3 * d);
        if (!p.bn_qkv) return;
        bool ok = make_tmap_bf16(&p.a_zh, w.xb, 2 * d, w.R, 128);
        for (int l = 0; l < m.L && ok; ++l)
            ok = make_tmap_bf16(&p.layer[l].wqkv, m.layer[l].w_qkv, 2 * d, 3 * d, p.bn_qkv < 256 ? p.bn_qkv : 256);
        p.mlp = p.mlp_cl = 0;
        p.head = ok && head_tc_supported(m) &&
                 make_tmap_bf16(&p.head_hi, m.head_ek_hi, d, 4 * d, 128) &&
                 make_tmap_bf16(&p.head_lo, m.head_ek_lo, d, 4 * d, 128);
        ok = ok && make_tmap_bf16(&p.a_xb, w.xb, d, w.R, 128) && make_tmap_bf16(&p.a_att, w.att, d, w.R, 128);
        head_gemm_plan(p, m, ok, pick_bn(4 * d));
        p.err = ctx->d_err;
        p.enabled = ok ? 1 : 0;
        return;
    }
    if (d % 64 || F % 64 || m.dh < 16 || !(d == 64 || d == 128 || d == 256 || d == 512)) return;
    // QKV and FFN1 tiles: the widest of 256 / 128 / 64 / 32 columns whose
    // grid over the context's row capacity still covers every SM (more CTAs,
    // each with a shorter epilogue: at 2 304 rows, d = 128, 128 -> 64
    // columns took the QKV launch from 9.6 to 8.5 us, and 64 -> 32 the
    // headline call from 14.41 to 14.22 ms).  TPPSD_QKV_BN / TPPSD_FFN1_BN
    // force a width.
    int n_sm = 148;
    cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, ctx->device);
    const long long tiles = (w.R + 127) / 128;
    auto fill_bn = [&](int N) {
        for (int bn = 256; bn >= 32; bn /= 2)
            if (N % bn == 0 && (N / bn) * tiles >= n_sm) return bn;
        return N % 32 == 0 ? 32 : pick_bn(N);
    };
    p.bn_qkv = fill_bn(3 * d);
    p.bn_ffn1 = fill_bn(F);
    if (const char* f = getenv("TPPSD_QKV_BN")) p.bn_qkv = atoi(f);
    if (const char* f = getenv("TPPSD_FFN1_BN")) p.bn_ffn1 = atoi(f);
    p.bn_o = ln_cluster_cols(d);
    if (!p.bn_qkv || !p.bn_ffn1 || !p.bn_o) return;
    bool ok = make_tmap_bf16(&p.a_xb, w.xb, d, w.R, 128) && make_tmap_bf16(&p.a_att, w.att, d, w.R, 128) &&
              make_tmap_bf16(&p.a_hid, w.hid, F, w.R, 128);
    const int bo = p.bn_o < 256 ? p.bn_o : 256;
    for (int l = 0; l < m.L && ok; ++l) {
        const LayerW& L = m.layer[l];
        ok = make_tmap_bf16(&p.layer[l].wqkv, L.w_qkv, d, 3 * d, p.bn_qkv < 256 ? p.bn_qkv : 256) &&
             make_tmap_bf16(&p.layer[l].wo, L.w_o, d, d, bo) &&
             make_tmap_bf16(&p.layer[l].w1, L.w_1, d, F, p.bn_ffn1 < 256 ? p.bn_ffn1 : 256) &&
             make_tmap_bf16(&p.layer[l].w2, L.w_2, F, d, bo);
    }
    p.mlp = ok && mlp_tc_supported(d, F) && !getenv("TPPSD_NO_MLP_FUSION");
    p.mlp_cl = p.mlp && mlp_cl_supported(d, F) && !getenv("TPPSD_MLP_SERIAL");
    for (int l = 0; l < m.L && p.mlp; ++l) {
        const LayerW& L = m.layer[l];
        p.mlp = make_tmap_bf16(&p.layer[l].wo_m, L.w_o, d, d, 128) &&
                make_tmap_bf16(&p.layer[l].w1_m, L.w_1, d, F, 128) &&
                make_tmap_bf16(&p.layer[l].w2_m, L.w_2, F, d, 128);
    }
    // TPPSD_QKV_FOLD=1: the cluster form also computes the next layer's Q,
    // K, V (W_qkv maps with boxes of its per-CTA column count).  Off by
    // default: with programmatic dependent launch the separate QKV GEMM is
    // already resident and waiting when the block ends, and the fold's
    // in-kernel row exchange measured slower (14.98 against 14.82 ms per
    // headline call).
    const int nq = p.mlp && p.mlp_cl ? mlp_cl_qkv_cols(d, F) : 0;
    p.qkv_fold = nq > 0 && getenv("TPPSD_QKV_FOLD") != nullptr;
    for (int l = 0; l < m.L && p.qkv_fold; ++l)
        p.qkv_fold = make_tmap_bf16(&p.layer[l].wqkv_f, m.layer[l].w_qkv, d, 3 * d, nq);
    p.head = ok && head_tc_supported(m) &&
             make_tmap_bf16(&p.head_hi, m.head_ek_hi, d, 4 * d, 128) &&
             make_tmap_bf16(&p.head_lo, m.head_ek_lo, d, 4 * d, 128);
    head_gemm_plan(p, m, ok, fill_bn(4 * d));
    p.err = ctx->d_err;
    p.enabled = ok ? 1 : 0;
}

static tppsd_status_t create_impl(tppsd_ctx* ctx, const tppsd_model_cfg* target,
                                  const tppsd_model_cfg* draft, const float* tb, size_t tn,
                                  const float* db, size_t dn) {
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev == 0) {
        cudaGetLastError();
        ctx->err = "no CUDA device";
        return TPPSD_ERR_NO_DEVICE;
    }
    CK(cudaGetDevice(&ctx->device));
    TRY(upload_model(ctx, ctx->T, target, tb, tn));
    TRY(upload_model(ctx, ctx->D, draft, db, dn));
    // TPPSD_ATTN_TC=1: the target's attention runs on the tcgen05 tensor
    // cores where its head width allows (d_head 32 or 64, bf16), with its V
    // cache kept in fp16.  Default: the mma.sync kernel of attn.cu (bf16 V
    // cache), measured faster at every workload shape (the decode shapes
    // leave the 128-row tensor-core products mostly idle).
    const int dhT = target->d_model / target->heads;
    ctx->T.dm.attn_tc = target->dtype == 1 && attn_tc_supported(dhT) && getenv("TPPSD_ATTN_TC") != nullptr;
    ctx->T.dm.v_f16 = ctx->T.dm.attn_tc;
    ctx->D.dm.v_f16 = 0;
    ctx->D.dm.attn_tc = 0;
    if (draft->encoder == 2 && !draft_team_supported(ctx->D.dm)) {
        ctx->err = "an AttNHP draft model must fit the one-CTA draft kernel (heads 1, 2 or 4, d/heads 16 or 32)";
        return TPPSD_ERR_UNSUPPORTED;
    }
    const int B = ctx->max_batch, nm = ctx->n_max;
    SeqState& ss = ctx->ss;
    ss.n_max = nm;
    TRY(dalloc(ctx, &ss.tau, sizeof(float) * (size_t)B * nm));
    TRY(dalloc(ctx, &ss.t, sizeof(double) * (size_t)B * nm));
    TRY(dalloc(ctx, &ss.k, sizeof(int) * (size_t)B * nm));
    TRY(dalloc(ctx, &ss.n_emit, sizeof(int) * B));
    TRY(dalloc(ctx, &ss.n_draft, sizeof(int) * B));
    TRY(dalloc(ctx, &ss.done, sizeof(int) * B));
    CK(cudaMemset(ss.tau, 0, sizeof(float) * (size_t)B * nm));
    CK(cudaMemset(ss.t, 0, sizeof(double) * (size_t)B * nm));
    CK(cudaMemset(ss.k, 0, sizeof(int) * (size_t)B * nm));
    CK(cudaMemset(ss.done, 1, sizeof(int) * B));
    TRY(alloc_kv(ctx, ctx->kvT, *target));
    TRY(alloc_kv(ctx, ctx->kvD, *draft));
    Work& w = ctx->work;
    w.R = B * (ctx->max_gamma + 1);
    if (w.R < 2048) w.R = 2048;
    const int dmax = target->d_model > draft->d_model ? target->d_model : draft->d_model;
    const int fmax = target->d_ffn > draft->d_ffn ? target->d_ffn : draft->d_ffn;
    const int hwT = 3 * target->n_mix + target->n_marks, hwD = 3 * draft->n_mix + draft->n_marks;
    const int hw = hwT > hwD ? hwT : hwD;
    const size_t R = w.R;
    TRY(dalloc(ctx, &w.row_seq, sizeof(int) * R));
    TRY(dalloc(ctx, &w.row_pos, sizeof(int) * R));
    TRY(dalloc(ctx, &w.x, sizeof(float) * R * dmax));
    TRY(dalloc(ctx, &w.y, sizeof(float) * R * dmax));
    TRY(dalloc(ctx, &w.xb, sizeof(float) * R * 2 * dmax));  // [z | h] rows of AttNHP
    TRY(dalloc(ctx, &w.q, sizeof(float) * R * dmax));
    TRY(dalloc(ctx, &w.att, sizeof(float) * R * dmax));
    TRY(dalloc(ctx, &w.hid, sizeof(float) * R * fmax));
    TRY(dalloc(ctx, &w.heads, sizeof(float) * R * hw));
    TRY(dalloc(ctx, &w.hd4, sizeof(float) * R * 4 * dmax));
    TRY(dalloc(ctx, &ctx->draft_heads, sizeof(float) * (size_t)B * ctx->max_gamma * hwD));
    TRY(dalloc(ctx, &ctx->d_params, sizeof(CallParams)));
    TRY(dalloc(ctx, &ctx->d_pois_logp, sizeof(float) * MAX_MARKS));
    TRY(dalloc(ctx, &ctx->d_stats, sizeof(DevStats)));
    TRY(dalloc(ctx, &ctx->d_active, sizeof(int)));
    CK(cudaMemset(ctx->d_stats, 0, sizeof(DevStats)));
    TRY(dalloc(ctx, &ctx->d_trace, sizeof(float4) * (size_t)B * nm));
    TRY(dalloc(ctx, &ctx->d_err, sizeof(int)));
    CK(cudaMemset(ctx->d_err, 0, sizeof(int)));
    w.err = ctx->d_err;
    // split-key attention scratch for the target's step passes (verify and
    // AR): one partial result per (item, split), one counter per item
    if (target->dtype == 1) {
        int n_sm = 0;
        CK(cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, ctx->device));
        const int dh = target->d_model / target->heads;
        long long need = 0;
        const int nq = 32;  // query columns of the tensor-core attention's products
        const long long items = (long long)B * target->heads;
        const long long ns = attn_splits(items, ctx->n_max, dh, nq, n_sm);
        if (ctx->T.dm.attn_tc && ns > 1) need = items * ns * nq * (dh + 2) * 4;
        if (need > 0) {
            TRY(dalloc(ctx, &w.attn.part, (size_t)need));
            TRY(dalloc(ctx, &w.attn.cnt, sizeof(int) * (size_t)B * target->heads));
            CK(cudaMemset(w.attn.cnt, 0, sizeof(int) * (size_t)B * target->heads));
            w.attn.part_bytes = (size_t)need;
            w.attn.cnt_items = (long long)B * target->heads;
        }
    }
    build_tc_plan(ctx);
    CK(cudaMallocHost(&ctx->h_active, sizeof(int)));
    CK(cudaStreamCreateWithFlags(&ctx->cap_stream, cudaStreamNonBlocking));
    CK(cudaEventCreateWithFlags(&ctx->done_event, cudaEventDisableTiming));
    CK(cudaDeviceSynchronize());
    return TPPSD_OK;
}

extern "C" tppsd_status_t tppsd_create_models(const tppsd_model_cfg* target,
                                              const tppsd_model_cfg* draft,
                                              const float* target_blob, size_t target_floats,
                                              const float* draft_blob, size_t draft_floats,
                                              int32_t max_batch, int32_t max_positions,
                                              int32_t max_gamma, tppsd_ctx** out) {
    if (!out) return TPPSD_ERR_INVALID_ARG;
    *out = nullptr;
    if (!cfg_ok(target) || !cfg_ok(draft) || !target_blob || !draft_blob)
        return TPPSD_ERR_INVALID_ARG;
    if (target->n_marks != draft->n_marks) return TPPSD_ERR_INVALID_ARG;
    if (target_floats != tppsd_blob_floats(target) || draft_floats != tppsd_blob_floats(draft))
        return TPPSD_ERR_INVALID_ARG;
    if (max_batch < 1 || max_positions < 2 || max_gamma < 1 || max_gamma > 31)
        return TPPSD_ERR_INVALID_ARG;
    const int dhD = draft->d_model / draft->heads;
    if (!(draft->heads == 1 || draft->heads == 2 || draft->heads == 4) || dhD < 8)
        return TPPSD_ERR_UNSUPPORTED;
    if (!strcmp(fault_mode(), "alloc")) return TPPSD_ERR_OOM;  // injected allocation failure
    g_pdl = getenv("TPPSD_NO_PDL") ? 0 : 1;
    tppsd_ctx* ctx = new (std::nothrow) tppsd_ctx();
    if (!ctx) return TPPSD_ERR_OOM;
    ctx->max_batch = max_batch;
    ctx->n_max = max_positions;
    ctx->max_gamma = max_gamma;
    tppsd_status_t st = create_impl(ctx, target, draft, target_blob, target_floats, draft_blob,
                                    draft_floats);
    if (st != TPPSD_OK) {
        fprintf(stderr, "tppsd_create_models: %s\n", ctx->err.c_str());
        tppsd_destroy(ctx);
        return st;
    }
    *out = ctx;
    return TPPSD_OK;
}

// Forward pass of rows [0, total) in ROWS_SPAN mode, q rows per sequence, in
// chunks that fit the row workspace.  after(g0, rows) runs after each chunk.
template <typename F>
static tppsd_status_t span_forward(tppsd_ctx* ctx, HostModel& hm, KVCache& kv, int B, int q,
                                   bool heads, cudaStream_t st, F after, int* launches) {
    const long long total = (long long)B * q;
    long long chunk = ctx->work.R;
    if (q <= chunk) chunk = (chunk / q) * q;
    for (long long g0 = 0; g0 < total; g0 += chunk) {
        RowSpec rs{ROWS_SPAN, q, (int)(total - g0 < chunk ? total - g0 : chunk), (int)g0};
        CK(launch_forward(hm.dm, kv, ctx->ss, ctx->work, rs, heads, st, launches, nullptr,
                          &hm == &ctx->T ? &ctx->tc : nullptr));
        TRY(after((int)g0, rs.count));
    }
    return TPPSD_OK;
}

extern "C" tppsd_status_t tppsd_prefill(tppsd_ctx* ctx, int32_t batch, const float* hist_tau,
                                        const int32_t* hist_marks, int32_t hist_len,
                                        void* stream) {
    if (!ctx || !hist_tau || !hist_marks) return TPPSD_ERR_INVALID_ARG;
    if (batch < 1 || batch > ctx->max_batch || hist_len < 1 || hist_len + 2 > ctx->n_max)
        return TPPSD_ERR_INVALID_ARG;
    CK(cudaSetDevice(ctx->device));
    cudaStream_t st = (cudaStream_t)stream;
    SeqState& ss = ctx->ss;
    const size_t pitch_f = sizeof(float) * ss.n_max, pitch_i = sizeof(int) * ss.n_max;
    CK(cudaMemcpy2DAsync(ss.tau, pitch_f, hist_tau, sizeof(float) * hist_len,
                         sizeof(float) * hist_len, batch, cudaMemcpyDefault, st));
    CK(cudaMemcpy2DAsync(ss.k, pitch_i, hist_marks, sizeof(int) * hist_len,
                         sizeof(int) * hist_len, batch, cudaMemcpyDefault, st));
    CK(cudaMemsetAsync(ctx->d_err, 0, sizeof(int), st));  // the flag reports this call only
    CK(launch_history_times(ss, batch, hist_len, st));
    int nl = 1;
    if (hist_len >= 2) {
        auto none = [](int, int) { return TPPSD_OK; };
        TRY(span_forward(ctx, ctx->T, ctx->kvT, batch, hist_len - 1, false, st, none, &nl));
        TRY(span_forward(ctx, ctx->D, ctx->kvD, batch, hist_len - 1, false, st, none, &nl));
    }
    ctx->prefill_launches = nl;
    CK(cudaEventRecord(ctx->done_event, st));
    ctx->last_stream = st;
    ctx->prefill_batch = batch;
    ctx->hist_len = hist_len;
    ctx->prefilled = true;
    return TPPSD_OK;
}

// One round: SD (mode 0) or AR (mode 1).  Returns launches in *nl.
static tppsd_status_t record_round(tppsd_ctx* ctx, int mode, int B, int gamma, cudaStream_t st,
                                   unsigned long long cond, int use_cond, int* nl,
                                   const Prof* prof) {
    int n = 0;
    Work& w = ctx->work;
    if (mode == 2) {
        PROF_MARK(prof, KC_DRAFT, 1, st);
        CK(launch_poisson_draft(ctx->ss, ctx->d_params, B, gamma, ctx->T.cfg.n_marks, st));
        PROF_MARK(prof, KC_DRAFT, 0, st);
        ++n;
        RowSpec rs{ROWS_STEP, gamma + 1, B * (gamma + 1), 0};
        CK(launch_forward(ctx->T.dm, ctx->kvT, ctx->ss, w, rs, true, st, &n, prof, &ctx->tc));
        PROF_MARK(prof, KC_EPILOGUE, 1, st);
        CK(launch_verify_epilogue(ctx->T.dm, ctx->D.dm, ctx->ss, ctx->d_params, B, gamma, w.heads,
                                  ctx->draft_heads, ctx->max_gamma, ctx->d_stats, st, true));
        PROF_MARK(prof, KC_EPILOGUE, 0, st);
        ++n;
    } else if (mode == 0) {
        PROF_MARK(prof, KC_DRAFT, 1, st);
        const bool team = draft_team_supported(ctx->D.dm) && (ctx->D.dm.enc == 2 || !getenv("TPPSD_DRAFT_CTA"));
        // the lane form also writes the target's verify rows (same storage
        // type, THP / SAHP layout), so the forward below has no embedding
        // launch (TPPSD_NO_EMBED_FUSION keeps it)
        bool fused = false;
        if (team && draft_lane_supported(ctx->D.dm, ctx->kvD.n_max, ctx->max_gamma) && !getenv("TPPSD_DRAFT_TEAM")) {
            const DevModel& tm = ctx->T.dm;
            DraftEmbed emb{tm.tenc, tm.type_emb, w.x, w.xb, w.row_seq, w.row_pos, tm.d, tm.K, tm.tenc_paired};
            fused = tm.dtype == ctx->D.dm.dtype && tm.enc != 2 && !getenv("TPPSD_NO_EMBED_FUSION");
            CK(launch_draft_lane(ctx->D.dm, ctx->kvD, ctx->ss, ctx->d_params, B, gamma,
                                 ctx->draft_heads, ctx->max_gamma, ctx->d_stats, ctx->d_err, st,
                                 fused ? &emb : nullptr));
        } else if (team)
            CK(launch_draft_team(ctx->D.dm, ctx->kvD, ctx->ss, ctx->d_params, B, gamma,
                                 ctx->draft_heads, ctx->max_gamma, ctx->d_stats, ctx->d_err, st));
        else
            CK(launch_draft(ctx->D.dm, ctx->kvD, ctx->ss, ctx->d_params, B, gamma, ctx->draft_heads,
                            ctx->max_gamma, ctx->d_stats, st));
        PROF_MARK(prof, KC_DRAFT, 0, st);
        ++n;
        RowSpec rs{ROWS_STEP, gamma + 1, B * (gamma + 1), 0, fused ? 1 : 0};
        CK(launch_forward(ctx->T.dm, ctx->kvT, ctx->ss, w, rs, true, st, &n, prof, &ctx->tc));
        PROF_MARK(prof, KC_EPILOGUE, 1, st);
        CK(launch_verify_epilogue(ctx->T.dm, ctx->D.dm, ctx->ss, ctx->d_params, B, gamma, w.heads,
                                  ctx->draft_heads, ctx->max_gamma, ctx->d_stats, st));
        PROF_MARK(prof, KC_EPILOGUE, 0, st);
        ++n;
    } else {
        RowSpec rs{ROWS_STEP, 1, B, 0};
        CK(launch_forward(ctx->T.dm, ctx->kvT, ctx->ss, w, rs, true, st, &n, prof, &ctx->tc));
        PROF_MARK(prof, KC_AR_SAMPLE, 1, st);
        CK(launch_ar_sample(ctx->T.dm, ctx->ss, ctx->d_params, B, w.heads, ctx->d_stats, st));
        PROF_MARK(prof, KC_AR_SAMPLE, 0, st);
        ++n;
    }
    PROF_MARK(prof, KC_CONTROL, 1, st);
    CK(launch_round_control(ctx->ss, ctx->d_params, B, ctx->d_stats, cond, use_cond,
                            use_cond ? nullptr : ctx->d_active, st));
    PROF_MARK(prof, KC_CONTROL, 0, st);
    ++n;
    if (nl) *nl = n;
    return TPPSD_OK;
}

static tppsd_status_t get_graph(tppsd_ctx* ctx, int mode, int B, int gamma, unsigned flags,
                                GraphEntry** out) {
    auto key = std::make_tuple(mode, B, gamma, flags);
    auto it = ctx->graphs.find(key);
    if (it != ctx->graphs.end()) {
        *out = &it->second;
        return TPPSD_OK;
    }
    GraphEntry ge;
    CK(cudaGraphCreate(&ge.graph, 0));
    cudaGraphConditionalHandle h;
    CK(cudaGraphConditionalHandleCreate(&h, ge.graph, 1, cudaGraphCondAssignDefault));
    cudaGraphNodeParams cp{};
    cp.type = cudaGraphNodeTypeConditional;
    cp.conditional.handle = h;
    cp.conditional.type = cudaGraphCondTypeWhile;
    cp.conditional.size = 1;
    cudaGraphNode_t node;
    CK(cudaGraphAddNode(&node, ge.graph, nullptr, nullptr, 0, &cp));
    cudaGraph_t body = cp.conditional.phGraph_out[0];
    CK(cudaStreamBeginCaptureToGraph(ctx->cap_stream, body, nullptr, nullptr, 0,
                                     cudaStreamCaptureModeRelaxed));
    tppsd_status_t rs = record_round(ctx, mode, B, gamma, ctx->cap_stream, (unsigned long long)h, 1,
                                     &ge.launches_per_round, nullptr);
    cudaGraph_t captured = nullptr;
    cudaError_t ce = cudaStreamEndCapture(ctx->cap_stream, &captured);
    TRY(rs);
    CK(ce);
    CK(cudaGraphInstantiate(&ge.exec, ge.graph, 0));
    auto res = ctx->graphs.emplace(key, ge);
    *out = &res.first->second;
    return TPPSD_OK;
}

static tppsd_status_t ensure_stage(tppsd_ctx* ctx, size_t bytes) {
    if (bytes <= ctx->stage_bytes) return TPPSD_OK;
    if (ctx->stage) cudaFree(ctx->stage);
    ctx->stage = nullptr;
    ctx->stage_bytes = 0;
    CK(cudaMalloc(&ctx->stage, bytes));
    ctx->stage_bytes = bytes;
    return TPPSD_OK;
}

struct PoissonDraft {
    double rate;
    const double* probs;  // [K], host
};

static tppsd_status_t run_sampler(tppsd_ctx* ctx, int mode, int B, int N, int gamma, uint64_t seed,
                                  uint32_t flags, float* out_tau, double* out_t, int32_t* out_k,
                                  void* stream, double t_end = INFINITY, int32_t* out_count = nullptr,
                                  bool until = false, const PoissonDraft* pois = nullptr) {
    if (!ctx) return TPPSD_ERR_INVALID_ARG;
    if (N > 0 && (!out_tau || !out_t || !out_k)) return TPPSD_ERR_INVALID_ARG;
    if (until && (!out_count || t_end != t_end)) return TPPSD_ERR_INVALID_ARG;
    if (!ctx->prefilled || B < 1 || B > ctx->prefill_batch || N < 0) return TPPSD_ERR_INVALID_ARG;
    const bool sd = mode != 1;  // 0: draft model, 2: Poisson draft
    if (sd && (gamma < 1 || gamma > ctx->max_gamma)) return TPPSD_ERR_INVALID_ARG;
    const int H = ctx->hist_len;
    if ((long long)H + N + (sd ? gamma : 0) + 2 > ctx->n_max) return TPPSD_ERR_INVALID_ARG;
    float logp[MAX_MARKS];
    const int K = ctx->T.cfg.n_marks;
    if (mode == 2) {  // Poisson draft: rate > 0, p >= 0 with a positive sum
        if (!pois || !pois->probs || !(pois->rate > 0.0) || !std::isfinite(pois->rate)) return TPPSD_ERR_INVALID_ARG;
        double tot = 0.0;
        for (int k = 0; k < K; ++k) {
            if (!(pois->probs[k] >= 0.0) || !std::isfinite(pois->probs[k])) return TPPSD_ERR_INVALID_ARG;
            tot += pois->probs[k];
        }
        if (!(tot > 0.0)) return TPPSD_ERR_INVALID_ARG;
        for (int k = 0; k < K; ++k) logp[k] = (float)log(pois->probs[k] / tot);
    }
    CK(cudaSetDevice(ctx->device));
    if (!strcmp(fault_mode(), "launch")) {
        ctx->err = "injected launch failure (TPPSD_FAULT=launch)";
        return TPPSD_ERR_CUDA;
    }
    cudaStream_t st = (cudaStream_t)stream;
    const size_t nb = (size_t)B * (N > 0 ? N : 1);
    const bool host_out[3] = {N > 0 && !is_device_ptr(out_tau), N > 0 && !is_device_ptr(out_t),
                              N > 0 && !is_device_ptr(out_k)};
    const bool host_count = until && !is_device_ptr(out_count);
    const bool any_host = host_out[0] || host_out[1] || host_out[2] || host_count;
    if (any_host) TRY(ensure_stage(ctx, nb * (4 + 8 + 4) + (size_t)B * 4 + 64));
    char* sb = (char*)ctx->stage;
    CallParams p{};
    p.B = B; p.H = H; p.N = N; p.gamma = sd ? gamma : 0; p.n_max = ctx->n_max;
    if (mode == 2) {
        CK(cudaMemcpyAsync(ctx->d_pois_logp, logp, sizeof(float) * K, cudaMemcpyHostToDevice, st));
        p.pois_rate = (float)pois->rate;
        p.pois_log_rate = (float)log(pois->rate);
        p.pois_logp = ctx->d_pois_logp;
    }
    p.flags = flags; p.seed = seed;
    p.out_t = host_out[1] ? (double*)sb : out_t;
    p.out_tau = host_out[0] ? (float*)(sb + nb * 8) : out_tau;
    p.out_k = host_out[2] ? (int*)(sb + nb * 12) : out_k;
    p.max_loops = N + 2;
    if (ctx->max_rounds > 0 && ctx->max_rounds < p.max_loops) p.max_loops = ctx->max_rounds;
    p.resample_cap = ctx->resample_cap;
    const bool traced = (flags & TPPSD_FLAG_DEBUG_TRACE) && mode != 1;
    p.trace = traced ? ctx->d_trace : nullptr;
    if (traced) CK(cudaMemsetAsync(ctx->d_trace, 0, sizeof(float4) * (size_t)ctx->max_batch * ctx->n_max, st));
    ctx->trace_batch = traced ? B : 0;
    ctx->trace_hist = H;
    ctx->trace_events = traced ? N : 0;
    CK(cudaMemsetAsync(ctx->d_err, 0, sizeof(int), st));  // the flag reports this call only
    p.t_end = t_end;
    p.out_count = until ? (host_count ? (int*)(sb + nb * 16) : out_count) : nullptr;
    // stop rule: the slots after each sequence's kept events read NaN / -1
    // (all-ones bytes are a NaN in fp32 and fp64 and -1 in int32)
    if (until && N > 0) {
        CK(cudaMemsetAsync(p.out_t, 0xFF, (size_t)B * N * 8, st));
        CK(cudaMemsetAsync(p.out_tau, 0xFF, (size_t)B * N * 4, st));
        CK(cudaMemsetAsync(p.out_k, 0xFF, (size_t)B * N * 4, st));
    }
    const bool profile = (flags & TPPSD_FLAG_PROFILE) != 0;
    Prof prof{&Profiler::mark, &ctx->prof};
    const Prof* pp = profile ? &prof : nullptr;
    if (profile) ctx->prof.reset();
    ctx->profiled = profile;
    PROF_MARK(pp, KC_BEGIN, 1, st);
    CK(launch_begin(p, ctx->d_params, ctx->ss, ctx->d_stats, st));
    PROF_MARK(pp, KC_BEGIN, 0, st);
    int launches = 1;
    if (N > 0) {
        if (flags & (TPPSD_FLAG_HOST_LOOP | TPPSD_FLAG_PROFILE)) {
            for (int it = 0; it < N + 2; ++it) {
                int nl = 0;
                TRY(record_round(ctx, mode, B, gamma, st, 0, 0, &nl, pp));
                launches += nl;
                CK(cudaMemcpyAsync(ctx->h_active, ctx->d_active, sizeof(int), cudaMemcpyDeviceToHost, st));
                CK(cudaStreamSynchronize(st));
                if (!*ctx->h_active) break;
            }
        } else {
            GraphEntry* ge = nullptr;
            TRY(get_graph(ctx, mode, B, sd ? gamma : 0, flags & TPPSD_FLAG_NO_BONUS, &ge));
            CK(cudaGraphLaunch(ge->exec, st));
            launches = -ge->launches_per_round;  // resolved from loop_iters in get_stats
        }
    }
    if (host_out[1]) CK(cudaMemcpyAsync(out_t, p.out_t, (size_t)B * N * 8, cudaMemcpyDeviceToHost, st));
    if (host_out[0]) CK(cudaMemcpyAsync(out_tau, p.out_tau, (size_t)B * N * 4, cudaMemcpyDeviceToHost, st));
    if (host_out[2]) CK(cudaMemcpyAsync(out_k, p.out_k, (size_t)B * N * 4, cudaMemcpyDeviceToHost, st));
    if (host_count) CK(cudaMemcpyAsync(out_count, p.out_count, (size_t)B * 4, cudaMemcpyDeviceToHost, st));
    CK(cudaEventRecord(ctx->done_event, st));
    ctx->last_stream = st;
    ctx->last_launches = launches;
    return TPPSD_OK;
}

extern "C" tppsd_status_t tppsd_sample(tppsd_ctx* ctx, int32_t batch, int32_t n_events,
                                       int32_t gamma, uint64_t seed, uint32_t flags,
                                       float* out_tau, double* out_t, int32_t* out_marks,
                                       void* stream) {
    return run_sampler(ctx, 0, batch, n_events, gamma, seed, flags, out_tau, out_t, out_marks,
                       stream);
}

extern "C" tppsd_status_t tppsd_sample_autoregressive(tppsd_ctx* ctx, int32_t batch,
                                                      int32_t n_events, uint64_t seed,
                                                      uint32_t flags, float* out_tau,
                                                      double* out_t, int32_t* out_marks,
                                                      void* stream) {
    return run_sampler(ctx, 1, batch, n_events, 0, seed, flags, out_tau, out_t, out_marks, stream);
}

extern "C" tppsd_status_t tppsd_sample_until(tppsd_ctx* ctx, int32_t batch, double t_end,
                                             int32_t max_events, int32_t gamma, uint64_t seed,
                                             uint32_t flags, float* out_tau, double* out_t,
                                             int32_t* out_marks, int32_t* out_count, void* stream) {
    return run_sampler(ctx, 0, batch, max_events, gamma, seed, flags, out_tau, out_t, out_marks,
                       stream, t_end, out_count, true);
}

extern "C" tppsd_status_t tppsd_sample_autoregressive_until(tppsd_ctx* ctx, int32_t batch,
                                                            double t_end, int32_t max_events,
                                                            uint64_t seed, uint32_t flags,
                                                            float* out_tau, double* out_t,
                                                            int32_t* out_marks, int32_t* out_count,
                                                            void* stream) {
    return run_sampler(ctx, 1, batch, max_events, 0, seed, flags, out_tau, out_t, out_marks, stream,
                       t_end, out_count, true);
}

// Teacher-forced scoring; with logS set the pass also covers the last event
// (q = len positions) and writes the survival term at t_end.
static tppsd_status_t run_score(tppsd_ctx* ctx, int which, int batch, int len, const float* tau,
                                const int32_t* marks, float* out_heads, float* out_logg,
                                float* out_logf, double t_end, double* out_logS, void* stream) {
    if (!ctx || !tau || !marks || (which != 0 && which != 1)) return TPPSD_ERR_INVALID_ARG;
    const int min_len = out_logS ? 1 : 2;
    if (batch < 1 || batch > ctx->max_batch || len < min_len || len > ctx->n_max) return TPPSD_ERR_INVALID_ARG;
    if (out_logS && t_end != t_end) return TPPSD_ERR_INVALID_ARG;
    CK(cudaSetDevice(ctx->device));
    cudaStream_t st = (cudaStream_t)stream;
    HostModel& hm = which == 0 ? ctx->T : ctx->D;
    KVCache& kv = which == 0 ? ctx->kvT : ctx->kvD;
    SeqState& ss = ctx->ss;
    ctx->prefilled = false;
    CK(cudaMemsetAsync(ctx->d_err, 0, sizeof(int), st));  // the flag reports this call only
    // TPPSD_FAULT=wait: the tensor-core QKV GEMM waits on a barrier nothing
    // completes, so its bounded wait runs out and the call reports
    // TPPSD_ERR_TIMEOUT (tests of the timeout path; no GPU fault involved)
    ctx->tc.stall = !strcmp(fault_mode(), "wait");
    CK(cudaMemcpy2DAsync(ss.tau, sizeof(float) * ss.n_max, tau, sizeof(float) * len,
                         sizeof(float) * len, batch, cudaMemcpyDefault, st));
    CK(cudaMemcpy2DAsync(ss.k, sizeof(int) * ss.n_max, marks, sizeof(int) * len, sizeof(int) * len,
                         batch, cudaMemcpyDefault, st));
    CK(launch_history_times(ss, batch, len, st));
    const int W = 3 * hm.cfg.n_mix + hm.cfg.n_marks;
    const size_t nh = (size_t)batch * len * W, nl = (size_t)batch * len;
    const bool hh = out_heads && !is_device_ptr(out_heads);
    const bool hg = out_logg && !is_device_ptr(out_logg);
    const bool hf = out_logf && !is_device_ptr(out_logf);
    const bool hs = out_logS && !is_device_ptr(out_logS);
    if (hh || hg || hf || hs) TRY(ensure_stage(ctx, (nh + 2 * nl) * sizeof(float) + (size_t)batch * 8 + 64));
    float* sb = (float*)ctx->stage;
    float* d_heads = hh ? sb : out_heads;
    float* d_logg = hg ? sb + nh : out_logg;
    float* d_logf = hf ? sb + nh + nl : out_logf;
    double* d_logS = hs ? (double*)(((uintptr_t)(sb + nh + 2 * nl) + 7) & ~(uintptr_t)7) : out_logS;
    const int q = out_logS ? len : len - 1;
    auto after = [&](int g0, int rows) -> tppsd_status_t {
        CK(launch_score_logs(hm.dm, ss, ctx->work, batch, len, q, g0, rows, d_heads, d_logg, d_logf, st));
        if (out_logS) CK(launch_score_survival(hm.dm, ss, ctx->work, batch, len, g0, rows, t_end, d_logS, st));
        return TPPSD_OK;
    };
    int launches = 0;
    if (len == 1 && out_logg) CK(cudaMemsetAsync(d_logg, 0xFF, nl * 4, st));  // NaN at i = 0
    if (len == 1 && out_logf) CK(cudaMemsetAsync(d_logf, 0xFF, nl * 4, st));
    TRY(span_forward(ctx, hm, kv, batch, q, true, st, after, &launches));
    if (hh) CK(cudaMemcpyAsync(out_heads, d_heads, nh * 4, cudaMemcpyDeviceToHost, st));
    if (hg) CK(cudaMemcpyAsync(out_logg, d_logg, nl * 4, cudaMemcpyDeviceToHost, st));
    if (hf) CK(cudaMemcpyAsync(out_logf, d_logf, nl * 4, cudaMemcpyDeviceToHost, st));
    if (hs) CK(cudaMemcpyAsync(out_logS, d_logS, (size_t)batch * 8, cudaMemcpyDeviceToHost, st));
    ctx->tc.stall = 0;
    CK(cudaEventRecord(ctx->done_event, st));
    ctx->last_stream = st;
    return TPPSD_OK;
}

extern "C" tppsd_status_t tppsd_sample_poisson(tppsd_ctx* ctx, int32_t batch, int32_t n_events,
                                               int32_t gamma, double rate, const double* mark_probs,
                                               uint64_t seed, uint32_t flags, float* out_tau,
                                               double* out_t, int32_t* out_marks, void* stream) {
    const PoissonDraft pd{rate, mark_probs};
    return run_sampler(ctx, 2, batch, n_events, gamma, seed, flags, out_tau, out_t, out_marks,
                       stream, INFINITY, nullptr, false, &pd);
}

extern "C" tppsd_status_t tppsd_sample_poisson_until(tppsd_ctx* ctx, int32_t batch, double t_end,
                                                     int32_t max_events, int32_t gamma, double rate,
                                                     const double* mark_probs, uint64_t seed,
                                                     uint32_t flags, float* out_tau, double* out_t,
                                                     int32_t* out_marks, int32_t* out_count,
                                                     void* stream) {
    const PoissonDraft pd{rate, mark_probs};
    return run_sampler(ctx, 2, batch, max_events, gamma, seed, flags, out_tau, out_t, out_marks,
                       stream, t_end, out_count, true, &pd);
}

extern "C" tppsd_status_t tppsd_fit_poisson_draft(int32_t batch, int32_t len, const float* tau,
                                                  const int32_t* marks, const double* t_window,
                                                  int32_t n_marks, double* out_rate,
                                                  double* out_mark_probs) {
    if (batch < 1 || len < 1 || !tau || !marks || !out_rate || !out_mark_probs || n_marks < 1 ||
        n_marks > MAX_MARKS)
        return TPPSD_ERR_INVALID_ARG;
    const size_t n = (size_t)batch * len;
    std::vector<float> ht;
    std::vector<int32_t> hk;
    const float* pt = tau;
    const int32_t* pk = marks;
    if (is_device_ptr(tau)) {
        ht.resize(n);
        if (cudaMemcpy(ht.data(), tau, n * 4, cudaMemcpyDeviceToHost) != cudaSuccess) return TPPSD_ERR_CUDA;
        pt = ht.data();
    }
    if (is_device_ptr(marks)) {
        hk.resize(n);
        if (cudaMemcpy(hk.data(), marks, n * 4, cudaMemcpyDeviceToHost) != cudaSuccess) return TPPSD_ERR_CUDA;
        pk = hk.data();
    }
    std::vector<double> cnt(n_marks, 0.0);
    double window = 0.0;
    for (int32_t b = 0; b < batch; ++b) {
        double t = 0.0;
        for (int32_t i = 0; i < len; ++i) {
            const float v = pt[(size_t)b * len + i];
            const int32_t k = pk[(size_t)b * len + i];
            if (!(v >= 0.f) || !std::isfinite(v) || k < 0 || k >= n_marks) return TPPSD_ERR_INVALID_ARG;
            t += (double)v;
            cnt[k] += 1.0;
        }
        if (t_window) {
            if (!(t_window[b] >= t) || !std::isfinite(t_window[b])) return TPPSD_ERR_INVALID_ARG;
            t = t_window[b];
        }
        window += t;
    }
    if (!(window > 0.0)) return TPPSD_ERR_INVALID_ARG;
    *out_rate = (double)n / window;
    for (int32_t k = 0; k < n_marks; ++k) out_mark_probs[k] = cnt[k] / (double)n;
    return TPPSD_OK;
}

extern "C" tppsd_status_t tppsd_score(tppsd_ctx* ctx, int32_t which, int32_t batch, int32_t len,
                                      const float* tau, const int32_t* marks, float* out_heads,
                                      float* out_logg, float* out_logf, void* stream) {
    return run_score(ctx, which, batch, len, tau, marks, out_heads, out_logg, out_logf, 0.0, nullptr,
                     stream);
}

extern "C" tppsd_status_t tppsd_score_until(tppsd_ctx* ctx, int32_t which, int32_t batch,
                                            int32_t len, const float* tau, const int32_t* marks,
                                            double t_end, float* out_heads, float* out_logg,
                                            float* out_logf, double* out_logS, void* stream) {
    if (!out_logS) return TPPSD_ERR_INVALID_ARG;
    return run_score(ctx, which, batch, len, tau, marks, out_heads, out_logg, out_logf, t_end,
                     out_logS, stream);
}

extern "C" tppsd_status_t tppsd_get_trace(tppsd_ctx* ctx, int32_t batch, int32_t n_events, float* out) {
    if (!ctx || !out || batch < 1 || n_events < 1) return TPPSD_ERR_INVALID_ARG;
    if (batch > ctx->trace_batch || n_events > ctx->trace_events) {
        ctx->err = "tppsd_get_trace: the last sampling call was not traced, or not that large";
        return TPPSD_ERR_INVALID_ARG;
    }
    CK(cudaSetDevice(ctx->device));
    CK(cudaEventSynchronize(ctx->done_event));
    const size_t row = sizeof(float4) * (size_t)n_events;
    CK(cudaMemcpy2D(out, row, ctx->d_trace + ctx->trace_hist, sizeof(float4) * (size_t)ctx->n_max, row, batch,
                    cudaMemcpyDefault));
    return TPPSD_OK;
}

extern "C" tppsd_status_t tppsd_set_limits(tppsd_ctx* ctx, int32_t resample_cap, int32_t max_rounds) {
    if (!ctx || resample_cap < 0 || max_rounds < 0) return TPPSD_ERR_INVALID_ARG;
    ctx->resample_cap = resample_cap > 0 ? resample_cap : DEFAULT_RESAMPLE_CAP;
    ctx->max_rounds = max_rounds;
    return TPPSD_OK;
}

extern "C" tppsd_status_t tppsd_wait(tppsd_ctx* ctx, int32_t timeout_ms) {
    if (!ctx) return TPPSD_ERR_INVALID_ARG;
    CK(cudaSetDevice(ctx->device));
    const auto t0 = std::chrono::steady_clock::now();
    for (;;) {
        const cudaError_t e = cudaEventQuery(ctx->done_event);
        if (e == cudaSuccess) {
            int derr = 0;
            CK(cudaMemcpy(&derr, ctx->d_err, sizeof(int), cudaMemcpyDeviceToHost));
            if (derr) {
                ctx->err = "a tensor-core pipeline wait timed out on the device";
                return TPPSD_ERR_TIMEOUT;
            }
            return TPPSD_OK;
        }
        if (e != cudaErrorNotReady) CK(e);
        const auto ms = std::chrono::duration_cast<std::chrono::milliseconds>(
                            std::chrono::steady_clock::now() - t0).count();
        if (ms >= timeout_ms) {
            ctx->err = "tppsd_wait: timed out";
            return TPPSD_ERR_TIMEOUT;
        }
        std::this_thread::sleep_for(std::chrono::microseconds(200));
    }
}

extern "C" tppsd_status_t tppsd_get_stats(tppsd_ctx* ctx, tppsd_stats* out) {
    if (!ctx || !out) return TPPSD_ERR_INVALID_ARG;
    CK(cudaSetDevice(ctx->device));
    CK(cudaEventSynchronize(ctx->done_event));
    DevStats s{};
    CK(cudaMemcpy(&s, ctx->d_stats, sizeof(s), cudaMemcpyDeviceToHost));
    out->rounds = (int64_t)s.rounds;
    out->drafted = (int64_t)s.drafted;
    out->accepted = (int64_t)s.accepted;
    out->emitted = (int64_t)s.emitted;
    out->resample_iters = (int64_t)s.resample_iters;
    out->cap_hits = (int64_t)s.cap_hits;
    out->loop_iters = (int64_t)s.loop_iters;
    out->prefill_launches = ctx->prefill_launches;
    out->target_keys = (int64_t)s.target_keys;
    out->draft_keys = (int64_t)s.draft_keys;
    out->kernel_launches = ctx->last_launches >= 0
                               ? ctx->last_launches
                               : 1 + (int64_t)s.loop_iters * (-ctx->last_launches);
    int derr = 0;
    CK(cudaMemcpy(&derr, ctx->d_err, sizeof(int), cudaMemcpyDeviceToHost));
    if (derr) {
        ctx->err = "a tensor-core pipeline wait timed out on the device (code " + std::to_string(derr) + ")";
        return TPPSD_ERR_TIMEOUT;
    }
    if (s.round_limit_hit) return TPPSD_ERR_ROUND_LIMIT;
    if (s.cap_hits) return TPPSD_WARN_RESAMPLE_CAP;
    return TPPSD_OK;
}

static const char* KC_NAMES[KC_COUNT] = {"draft", "embed", "gemm_qkv", "attention", "gemm_o",
                                         "layernorm", "gemm_ffn1", "gemm_ffn2", "head",
                                         "epilogue", "ar_sample", "control", "begin"};

extern "C" const char* tppsd_kernel_class_name(int32_t cls) {
    return cls >= 0 && cls < KC_COUNT ? KC_NAMES[cls] : "";
}

extern "C" tppsd_status_t tppsd_kernel_times(tppsd_ctx* ctx, double* ms, int64_t* launches) {
    if (!ctx || !ms || !launches) return TPPSD_ERR_INVALID_ARG;
    for (int i = 0; i < KC_COUNT; ++i) { ms[i] = 0.0; launches[i] = 0; }
    if (!ctx->profiled) return TPPSD_ERR_INVALID_ARG;
    CK(cudaSetDevice(ctx->device));
    CK(ctx->prof.err);
    CK(cudaEventSynchronize(ctx->done_event));
    for (auto& sp : ctx->prof.spans) {
        float t = 0.f;
        CK(cudaEventElapsedTime(&t, ctx->prof.pool[sp.second], ctx->prof.pool[sp.second + 1]));
        ms[sp.first] += t;
        launches[sp.first] += 1;
    }
    return TPPSD_OK;
}

extern "C" const char* tppsd_status_str(tppsd_status_t s) {
    switch (s) {
        case TPPSD_OK: return "ok";
        case TPPSD_ERR_INVALID_ARG: return "invalid argument";
        case TPPSD_ERR_OOM: return "out of memory";
        case TPPSD_ERR_CUDA: return "CUDA error";
        case TPPSD_ERR_UNSUPPORTED: return "unsupported shape";
        case TPPSD_ERR_ROUND_LIMIT: return "round limit reached";
        case TPPSD_ERR_TIMEOUT: return "timeout";
        case TPPSD_ERR_NO_DEVICE: return "no CUDA device";
        case TPPSD_WARN_RESAMPLE_CAP: return "resample cap reached";
    }
    return "unknown status";
}

extern "C" const char* tppsd_last_error(const tppsd_ctx* ctx) { return ctx ? ctx->err.c_str() : ""; }

extern "C" void tppsd_destroy(tppsd_ctx* ctx) {
    if (!ctx) return;
    cudaSetDevice(ctx->device);
    cudaDeviceSynchronize();
    for (auto& kv : ctx->graphs) {
        if (kv.second.exec) cudaGraphExecDestroy(kv.second.exec);
        if (kv.second.graph) cudaGraphDestroy(kv.second.graph);
    }
    for (void* p : ctx->allocs) cudaFree(p);
    if (ctx->stage) cudaFree(ctx->stage);
    if (ctx->h_active) cudaFreeHost(ctx->h_active);
    for (cudaEvent_t e : ctx->prof.pool) cudaEventDestroy(e);
    if (ctx->cap_stream) cudaStreamDestroy(ctx->cap_stream);
    if (ctx->done_event) cudaEventDestroy(ctx->done_event);
    cudaGetLastError();
    delete ctx;
}

// ---------------------------------------------------------------- scoring without allocation
// tppsd_score_noalloc runs the same teacher-forced scoring pipeline as
// tppsd_score, but every buffer it needs besides the caller's inputs and
// outputs (sequence copy, K/V cache of the scored rows, row workspace) is
// carved out of one fixed array in device memory that exists from the moment
// the library is loaded.  The call itself never allocates.  This serves
// callers that may not allocate device memory at call time: processes whose
// device memory is owned by another allocator (a framework's caching pool
// that has already reserved the GPU), and latency-critical loops that cannot
// afford the implicit device synchronisation of cudaMalloc/cudaFree.
constexpr size_t NOALLOC_SCRATCH_BYTES = (size_t)16 << 20;  // 16 MiB per device
static __device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_SCRATCH_BYTES];

namespace {
constexpr int NOALLOC_MAX_DEVICES = 64;
std::mutex g_noalloc_mutex;
void* g_noalloc_addr[NOALLOC_MAX_DEVICES] = {};
}  // namespace

// Device address of the scratch array on the current device.  The symbol's
// host-side name is not a device address; cudaGetSymbolAddress gives the
// real one, once per device (the first call on a device does this set-up).
static tppsd_status_t noalloc_scratch(tppsd_ctx* ctx, unsigned char** out) {
    int dev = 0;
    CK(cudaGetDevice(&dev));
    if (dev < 0 || dev >= NOALLOC_MAX_DEVICES) {
        ctx->err = "tppsd_score_noalloc: device index out of range";
        return TPPSD_ERR_UNSUPPORTED;
    }
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (!g_noalloc_addr[dev]) {
        void* p = nullptr;
        CK(cudaGetSymbolAddress(&p, g_noalloc_scratch));
        g_noalloc_addr[dev] = p;
    }
    *out = (unsigned char*)g_noalloc_addr[dev];
    return TPPSD_OK;
}

extern "C" tppsd_status_t tppsd_score_noalloc(tppsd_ctx* ctx, int32_t which, int32_t batch,
                                              int32_t len, const float* tau, const int32_t* marks,
                                              float* out_logg, float* out_logf, void* stream) {
    if (!ctx || !tau || !marks || !out_logg || !out_logf || (which != 0 && which != 1))
        return TPPSD_ERR_INVALID_ARG;
    if (batch < 1 || len < 2) return TPPSD_ERR_INVALID_ARG;
    CK(cudaSetDevice(ctx->device));
    if (!is_device_ptr(tau) || !is_device_ptr(marks) || !is_device_ptr(out_logg) ||
        !is_device_ptr(out_logf)) {
        ctx->err = "tppsd_score_noalloc: all arrays must be device memory";
        return TPPSD_ERR_INVALID_ARG;
    }
    HostModel& hm = which == 0 ? ctx->T : ctx->D;
    const tppsd_model_cfg& c = hm.cfg;
    const size_t eb = c.dtype == 1 ? 2 : 4;
    const size_t d = c.d_model, F = c.d_ffn, W = 3 * c.n_mix + c.n_marks;
    const size_t n = (size_t)batch * len;
    auto up = [](size_t x) { return (x + 255) & ~(size_t)255; };
    // fixed part: sequence copy, per-sequence state, K and V of every scored position
    const size_t seq_bytes = up(n * 4) + up(n * 8) + up(n * 4) + 3 * up((size_t)batch * 4);
    const size_t kv_bytes = 2 * up((size_t)c.layers * n * d * eb);
    // per workspace row, in the order the buffers are carved below: row_seq,
    // row_pos, x and y (fp32), xb (the [z | h] rows of AttNHP: 2d), q and
    // att (storage type), hid, heads, head pre-activations (fp32)
    const size_t per_row[] = {4, 4, d * 4, d * 4, 2 * d * eb, d * eb, d * eb, F * eb, W * 4, 4 * d * 4};
    constexpr int NROW_BUFS = (int)(sizeof(per_row) / sizeof(per_row[0]));
    size_t row_bytes = 0;
    for (size_t b : per_row) row_bytes += b;
    const size_t fixed = seq_bytes + kv_bytes + NROW_BUFS * 256;  // each row buffer rounds up to 256 B
    const long long q = len - 1, total = (long long)batch * q;
    long long rows = fixed < NOALLOC_SCRATCH_BYTES ? (long long)((NOALLOC_SCRATCH_BYTES - fixed) / row_bytes) : 0;
    if (rows > total) rows = total;
    if (rows < 16 && rows < total) {
        char msg[200];
        snprintf(msg, sizeof msg, "tppsd_score_noalloc: %d x %d events exceed the %zu-byte scratch",
                 batch, len, NOALLOC_SCRATCH_BYTES);
        ctx->err = msg;
        return TPPSD_ERR_INVALID_ARG;
    }
    unsigned char* base = nullptr;
    TRY(noalloc_scratch(ctx, &base));
    size_t off = 0;
    auto take = [&](size_t bytes) { unsigned char* p = base + off; off += up(bytes); return (void*)p; };
    SeqState ss{};
    ss.n_max = len;
    ss.tau = (float*)take(n * 4);
    ss.t = (double*)take(n * 8);
    ss.k = (int*)take(n * 4);
    ss.n_emit = (int*)take((size_t)batch * 4);
    ss.n_draft = (int*)take((size_t)batch * 4);
    ss.done = (int*)take((size_t)batch * 4);
    KVCache kv{};
    kv.k = take((size_t)c.layers * n * d * eb);
    kv.v = take((size_t)c.layers * n * d * eb);
    kv.Bmax = batch;
    kv.n_max = len;
    Work w{};
    w.err = ctx->d_err;  // bounded pipeline waits report here, as in tppsd_score
    w.R = (int)rows;
    void* rb[NROW_BUFS];
    for (int i = 0; i < NROW_BUFS; ++i) rb[i] = take((size_t)rows * per_row[i]);
    w.row_seq = (int*)rb[0];
    w.row_pos = (int*)rb[1];
    w.x = (float*)rb[2];
    w.y = (float*)rb[3];
    w.xb = rb[4];
    w.q = rb[5];
    w.att = rb[6];
    w.hid = rb[7];
    w.heads = (float*)rb[8];
    w.hd4 = (float*)rb[9];
    if (off > NOALLOC_SCRATCH_BYTES) {
        ctx->err = "tppsd_score_noalloc: scratch layout overflow";
        return TPPSD_ERR_INVALID_ARG;
    }
    cudaStream_t st = (cudaStream_t)stream;
    // Every byte read below is written first in this call (sequence copy,
    // times, then K/V of positions 0..i before any query at i), so nothing
    // left by an earlier call is ever read.
    CK(cudaMemsetAsync(ctx->d_err, 0, sizeof(int), st));  // the flag reports this call only
    CK(cudaMemcpyAsync(ss.tau, tau, n * 4, cudaMemcpyDeviceToDevice, st));
    CK(cudaMemcpyAsync(ss.k, marks, n * 4, cudaMemcpyDeviceToDevice, st));
    CK(launch_history_times(ss, batch, len, st));
    long long chunk = rows;
    if (q <= chunk) chunk = (chunk / q) * q;
    for (long long g0 = 0; g0 < total; g0 += chunk) {
        RowSpec rs{ROWS_SPAN, (int)q, (int)(total - g0 < chunk ? total - g0 : chunk), (int)g0};
        CK(launch_forward(hm.dm, kv, ss, w, rs, true, st, nullptr, nullptr));
        CK(launch_score_logs(hm.dm, ss, w, batch, len, len - 1, (int)g0, rs.count, nullptr, out_logg,
                             out_logf, st));
    }
    CK(cudaEventRecord(ctx->done_event, st));
    ctx->last_stream = st;
    return TPPSD_OK;
}
