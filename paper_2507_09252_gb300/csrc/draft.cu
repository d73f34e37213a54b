// Draft loop of TPP-SD (Sec. 4.3 "Drafting", Alg. 1): one warp per sequence.
//
// Each round a warp catches its draft cache up to the last emitted event and
// then drafts gamma events: head of the draft model -> direct sample
// (z ~ Cat(w), eps ~ N(0,1), tau = exp(mu_z + sigma_z eps); k ~ f, Sec. 4.2)
// -> encode the drafted event -> next head.  A d-vector is spread over the
// warp (element i in lane i % 32, register i / 32), so a matrix-vector
// product broadcasts each input element by shuffle against weights stored
// [in][out]; nothing waits on a block barrier.  The draft model (transposed
// copy) is staged in shared memory once per CTA when it fits, and each
// warp's draft KV cache is loaded into shared memory once per round (and
// written through to HBM), so all gamma steps read weights and keys on chip.
#include <math.h>

#include "common.cuh"
#include "engine.h"
#include "tc_ptx.cuh"

namespace tppsd {

constexpr unsigned FULL = 0xffffffffu;

struct DraftWArgs {
    DevModel m;
    KVCache kv;
    SeqState ss;
    const CallParams* P;
    DevStats* st;
    float* heads;      // [Bmax][gamma_max][W]
    int gamma, gamma_max;
    int w_smem;        // stage the transposed model in shared memory
    int wpc;           // warps (sequences) per CTA
    int w_bytes;       // staged model bytes (16-aligned), 0 if not staged
    int warp_bytes;    // per-warp shared bytes (KV if resident + scratch)
    int* err;          // set if the KV bulk load does not complete
};

// DH consecutive storage-type values -> fp32, with 16-byte loads.
template <typename T, int DH>
__device__ __forceinline__ void load_row16(const T* p, float (&out)[DH]) {
    constexpr int PER = 16 / sizeof(T);
    static_assert(DH % PER == 0, "row must be a whole number of 16-byte chunks");
#pragma unroll
    for (int c = 0; c < DH / PER; ++c) {
        const uint4 w = reinterpret_cast<const uint4*>(p)[c];
        if constexpr (sizeof(T) == 2) {
            const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&w);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 f = __bfloat1622float2(h[i]);
                out[c * 8 + 2 * i] = f.x;
                out[c * 8 + 2 * i + 1] = f.y;
            }
        } else {
            out[c * 4 + 0] = __uint_as_float(w.x);
            out[c * 4 + 1] = __uint_as_float(w.y);
            out[c * 4 + 2] = __uint_as_float(w.z);
            out[c * 4 + 3] = __uint_as_float(w.w);
        }
    }
}

template <int N> struct Regs { static constexpr int n = (N + 31) / 32; };

// element i of a warp-distributed vector
template <int NR>
__device__ __forceinline__ float bcast(const float (&v)[NR], int i) {
    return __shfl_sync(FULL, v[i >> 5], i & 31);
}

// y[o] = sum_{i<IN} WT[i][o] x[OFF + i] + b[o], OUT outputs (o = lane + 32 a).
template <int IN, int OFF, int OUT, typename TW, int NX>
__device__ __forceinline__ void wmv(const TW* __restrict__ WT, const float* __restrict__ b,
                                    const float (&x)[NX], float (&y)[Regs<OUT>::n], int lane) {
    constexpr int NY = Regs<OUT>::n;
#pragma unroll
    for (int a = 0; a < NY; ++a) {
        const int o = lane + 32 * a;
        y[a] = (b && o < OUT) ? b[o] : 0.f;
    }
    // input element ii = 32 r + j lives in register r of lane j: r is a
    // compile-time index, j a run-time one
#pragma unroll
    for (int r = OFF / 32; r < (OFF + IN + 31) / 32; ++r) {
#pragma unroll 4
        for (int j = 0; j < 32; ++j) {
            const int ii = 32 * r + j;
            if (ii < OFF || ii >= OFF + IN) continue;
            const float xi = __shfl_sync(FULL, x[r], j);
            const TW* row = WT + (size_t)(ii - OFF) * OUT;
#pragma unroll
            for (int a = 0; a < NY; ++a) {
                const int o = lane + 32 * a;
                if (o < OUT) y[a] = fmaf(St<TW>::ld(row + o), xi, y[a]);
            }
        }
    }
}

// Same with a run-time output count (head outputs M, K), at most 32*NY.
template <int IN, int OFF, int NY, int NX>
__device__ __forceinline__ void wmv_rt(const float* __restrict__ WT, const float* __restrict__ b,
                                       int OUT, const float (&x)[NX], float (&y)[NY], int lane) {
#pragma unroll
    for (int a = 0; a < NY; ++a) {
        const int o = lane + 32 * a;
        y[a] = o < OUT ? b[o] : 0.f;
    }
#pragma unroll
    for (int r = OFF / 32; r < (OFF + IN + 31) / 32; ++r) {
#pragma unroll 4
        for (int j = 0; j < 32; ++j) {
            const int ii = 32 * r + j;
            if (ii < OFF || ii >= OFF + IN) continue;
            const float xi = __shfl_sync(FULL, x[r], j);
            const float* row = WT + (size_t)(ii - OFF) * OUT;
#pragma unroll
            for (int a = 0; a < NY; ++a) {
                const int o = lane + 32 * a;
                if (o < OUT) y[a] = fmaf(row[o], xi, y[a]);
            }
        }
    }
}

template <int D, int NR>
__device__ __forceinline__ void wlayernorm(float (&x)[NR], const float* g, const float* b, int lane) {
    float s = 0.f;
#pragma unroll
    for (int a = 0; a < NR; ++a) if (lane + 32 * a < D) s += x[a];
    const float mean = warp_sum(s) / D;
    float v = 0.f;
#pragma unroll
    for (int a = 0; a < NR; ++a) if (lane + 32 * a < D) v += (x[a] - mean) * (x[a] - mean);
    const float inv = 1.0f / sqrtf(warp_sum(v) / D + LN_EPS);
#pragma unroll
    for (int a = 0; a < NR; ++a) {
        const int i = lane + 32 * a;
        x[a] = i < D ? (x[a] - mean) * inv * g[i] + b[i] : 0.f;
    }
}

// In-warp log-softmax of NY-register values with n live entries.
template <int NY>
__device__ __forceinline__ void wlogsoftmax(float (&v)[NY], int n, int lane) {
    float mx = -INFINITY;
#pragma unroll
    for (int a = 0; a < NY; ++a) if (lane + 32 * a < n) mx = fmaxf(mx, v[a]);
    mx = warp_max(mx);
    float s = 0.f;
#pragma unroll
    for (int a = 0; a < NY; ++a) if (lane + 32 * a < n) s += expf(v[a] - mx);
    const float lz = mx + logf(warp_sum(s));
#pragma unroll
    for (int a = 0; a < NY; ++a) v[a] -= lz;
}

// Smallest index whose running sum of exp(logp) reaches u * total, for a
// warp-distributed vector (inclusive warp scan per register).
template <int NY>
__device__ __forceinline__ int wpick(const float (&logp)[NY], int n, float u, int lane) {
    float p[NY], tot = 0.f;
#pragma unroll
    for (int a = 0; a < NY; ++a) {
        p[a] = lane + 32 * a < n ? expf(logp[a]) : 0.f;
        tot += p[a];
    }
    tot = warp_sum(tot);
    const float target = u * tot;
    float base = 0.f;
#pragma unroll
    for (int a = 0; a < NY; ++a) {
        float c = p[a];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const float t = __shfl_up_sync(FULL, c, o);
            if (lane >= o) c += t;
        }
        const unsigned hit = __ballot_sync(FULL, lane + 32 * a < n && base + c >= target);
        if (hit) return 32 * a + __ffs(hit) - 1;
        base += __shfl_sync(FULL, c, 31);
    }
    return n - 1;
}

// value of register-distributed v at run-time index i
template <int NY>
__device__ __forceinline__ float wget(const float (&v)[NY], int i) {
    float r = 0.f;
#pragma unroll
    for (int a = 0; a < NY; ++a) if ((i >> 5) == a) r = v[a];
    return __shfl_sync(FULL, r, i & 31);
}

template <typename T, int D, int F, int DH, bool KVS>
struct DraftWarp {
    static constexpr int NH = D / DH;
    static constexpr int R1 = Regs<D>::n;       // d-vector registers
    static constexpr int R3 = Regs<3 * D>::n;
    static constexpr int RF = Regs<F>::n;
    static constexpr int RM = 2;                // M <= 64
    static constexpr int RK = 8;                // K <= 256

    const DevModelT& m;   // pointer table in shared memory (rebased when staged)
    const DraftWArgs& a;
    int s, lane, L, M, K, n_max;
    T* kv_s;                                    // per-warp resident KV: [L][2][NH][n_max][DH]
    float* scratch;                             // per-warp D floats
    uint64_t* bar;                              // per-warp mbarrier of the KV bulk load

    __device__ T* kslot(int l, int which, int h, int pos) const {
        if (KVS) return kv_s + ((((size_t)l * 2 + which) * NH + h) * n_max + pos) * DH;
        T* base = (T*)(which ? a.kv.v : a.kv.k);
        return base + ((((size_t)l * a.kv.Bmax + s) * NH + h) * (size_t)a.kv.n_max + pos) * DH;
    }

    // Positions 0..nd-1 of every (layer, K/V, head) are one contiguous block
    // in HBM: one bulk copy each into shared memory, completing on the
    // warp's mbarrier.
    __device__ void load_kv(int nd) {
        if (!KVS || nd <= 0) return;
        const uint32_t bytes = (uint32_t)nd * DH * sizeof(T);
        if (lane == 0) {
            mbar_init(bar, 1);
            mbar_fence_init();
            mbar_arrive_expect_tx(bar, bytes * (uint32_t)(L * 2 * NH));
            for (int l = 0; l < L; ++l)
                for (int w = 0; w < 2; ++w)
                    for (int h = 0; h < NH; ++h) {
                        const T* src = (const T*)(w ? a.kv.v : a.kv.k) +
                                       ((((size_t)l * a.kv.Bmax + s) * NH + h) * (size_t)a.kv.n_max) * DH;
                        bulk_load(kslot(l, w, h, 0), src, bytes, bar);
                    }
        }
        __syncwarp();
        mbar_wait(bar, 0, a.err, 11);
        __syncwarp();
    }

    __device__ void store_kv(int l, int which, int h, int pos, int e, float v) const {
        St<T>::st(kslot(l, which, h, pos) + e, v);
        if (KVS) {
            T* g = (T*)(which ? a.kv.v : a.kv.k) +
                   ((((size_t)l * a.kv.Bmax + s) * NH + h) * (size_t)a.kv.n_max + pos) * DH;
            St<T>::st(g + e, v);
        }
    }

    // attention of one query (q, distributed) over keys 0..p of layer l
    __device__ void attend(int l, int p, const float (&qkv)[R3], float (&att)[R1]) {
        const float scale = 1.0f / sqrtf((float)DH);
#pragma unroll
        for (int h = 0; h < NH; ++h) {
            float q[DH];
#pragma unroll
            for (int e = 0; e < DH; ++e) q[e] = bcast(qkv, h * DH + e) * scale;
            float mm = -INFINITY, ll = 0.f, o[DH];
#pragma unroll
            for (int e = 0; e < DH; ++e) o[e] = 0.f;
            const T* kb = kslot(l, 0, h, 0);
            const T* vb = kslot(l, 1, h, 0);
            for (int j = lane; j <= p; j += 32) {
                float kr[DH], vr[DH];
                load_row16<T, DH>(kb + (size_t)j * DH, kr);
                load_row16<T, DH>(vb + (size_t)j * DH, vr);
                float sc = 0.f;
#pragma unroll
                for (int e = 0; e < DH; ++e) sc = fmaf(q[e], kr[e], sc);
                const float mn = fmaxf(mm, sc), corr = expf(mm - mn), pj = expf(sc - mn);
                ll = ll * corr + pj;
#pragma unroll
                for (int e = 0; e < DH; ++e) o[e] = fmaf(pj, vr[e], o[e] * corr);
                mm = mn;
            }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                const float m2 = __shfl_xor_sync(FULL, mm, off);
                const float l2 = __shfl_xor_sync(FULL, ll, off);
                float a2 = 0.f, b2 = 0.f;
                if (m2 != -INFINITY || mm != -INFINITY) {
                    const float mn = fmaxf(mm, m2);
                    a2 = mm == -INFINITY ? 0.f : expf(mm - mn);
                    b2 = m2 == -INFINITY ? 0.f : expf(m2 - mn);
                    mm = mn;
                }
                ll = ll * a2 + l2 * b2;
#pragma unroll
                for (int e = 0; e < DH; ++e) {
                    const float o2 = __shfl_xor_sync(FULL, o[e], off);
                    o[e] = o[e] * a2 + o2 * b2;
                }
            }
            if (lane == 0) {
                const float inv = 1.0f / ll;
#pragma unroll
                for (int e = 0; e < DH; ++e) scratch[h * DH + e] = o[e] * inv;
            }
        }
        __syncwarp();
#pragma unroll
        for (int r = 0; r < R1; ++r) {
            const int i = lane + 32 * r;
            att[r] = i < D ? St<T>::rnd(scratch[i]) : 0.f;
        }
        __syncwarp();
    }

    // Encode the event at position p; leaves the final hidden state in x.
    __device__ void encode(int p, float (&x)[R1]) {
        const SeqState& ss = a.ss;
        const size_t so = (size_t)s * ss.n_max + p;
        const double t = ss.t[so];
        const int k = min(max(ss.k[so], 0), K - 1);
#pragma unroll
        for (int r = 0; r < R1; ++r) {
            const int i = lane + 32 * r;
            if (i < D) {
                const double ang = t * m.omega[i >> 1];
                const double red = fma(-6.283185307179586476925, rint(ang * 0.15915494309189533577), ang);
                float sv, cv;
                sincosf((float)red, &sv, &cv);
                x[r] = ((i & 1) ? cv : sv) + m.type_emb[(size_t)k * D + i];
            } else {
                x[r] = 0.f;
            }
        }
        for (int l = 0; l < L; ++l) {
            const LayerW& W = m.layer[l];
            float xin[R1], qkv[R3], att[R1], y[R1], hid[RF];
#pragma unroll
            for (int r = 0; r < R1; ++r) xin[r] = St<T>::rnd(x[r]);
            wmv<D, 0, 3 * D, T>((const T*)W.w_qkv, W.b_qkv, xin, qkv, lane);
#pragma unroll
            for (int r = 0; r < R3; ++r) {
                const int o = lane + 32 * r;
                qkv[r] = St<T>::rnd(qkv[r]);
                if (o >= D && o < 3 * D) {
                    const int which = o < 2 * D ? 0 : 1, c = o - D - which * D;
                    store_kv(l, which, c / DH, p, c % DH, qkv[r]);
                }
            }
            __syncwarp();
            attend(l, p, qkv, att);
            wmv<D, 0, D, T>((const T*)W.w_o, W.b_o, att, y, lane);
#pragma unroll
            for (int r = 0; r < R1; ++r) x[r] += y[r];
            wlayernorm<D>(x, W.ln1_g, W.ln1_b, lane);
#pragma unroll
            for (int r = 0; r < R1; ++r) xin[r] = St<T>::rnd(x[r]);
            wmv<D, 0, F, T>((const T*)W.w_1, W.b_1, xin, hid, lane);
#pragma unroll
            for (int r = 0; r < RF; ++r) hid[r] = St<T>::rnd(fmaxf(hid[r], 0.f));
            wmv<F, 0, D, T>((const T*)W.w_2, W.b_2, hid, y, lane);
#pragma unroll
            for (int r = 0; r < R1; ++r) x[r] += y[r];
            wlayernorm<D>(x, W.ln2_g, W.ln2_b, lane);
        }
    }

    // Head of Sec. 4.2 from x: lw (log w), mu, sg (log sigma), lk (log f).
    __device__ void head(const float (&x)[R1], float (&lw)[RM], float (&mu)[RM], float (&sg)[RM],
                         float (&lk)[RK]) {
        const HeadW& H = m.head;
        float e[R3], av[R1];
        wmv<D, 0, 3 * D, float>(H.E, nullptr, x, e, lane);
        wmv<D, 0, D, float>(H.v_k1, H.b_k1, x, av, lane);
#pragma unroll
        for (int r = 0; r < R1; ++r) av[r] = tanhf(av[r]);
        wmv_rt<D, 0, RM>(H.v_w, H.b_w, M, e, lw, lane);
        wmv_rt<D, D, RM>(H.v_mu, H.b_mu, M, e, mu, lane);
        wmv_rt<D, 2 * D, RM>(H.v_s, H.b_s, M, e, sg, lane);
        wmv_rt<D, 0, RK>(H.v_k2, H.b_k2, K, av, lk, lane);
        wlogsoftmax<RM>(lw, M, lane);
        wlogsoftmax<RK>(lk, K, lane);
    }
};

template <typename T, int D, int F, int DH, bool KVS>
__global__ void __launch_bounds__(128) k_draft_warp(DraftWArgs a) {
    extern __shared__ __align__(16) char smem[];
    __shared__ DevModelT m;  // one pointer table per CTA, read by every thread
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (a.w_smem) {
        const int4* src = (const int4*)a.m.t.base;
        int4* dst = (int4*)smem;
        for (size_t i = threadIdx.x; i < a.m.t.bytes / 16; i += blockDim.x) dst[i] = src[i];
    }
    if (threadIdx.x == 0) {
        m = a.m.t;
        if (a.w_smem) {
            const char* ob = a.m.t.base;
            auto rb = [&](const void* p) { return (const char*)smem + ((const char*)p - ob); };
            m.type_emb = (const float*)rb(m.type_emb);
            m.omega = (const double*)rb(m.omega);
            for (int l = 0; l < a.m.L; ++l) {
                LayerW& L = m.layer[l];
                L.w_qkv = rb(L.w_qkv); L.b_qkv = (const float*)rb(L.b_qkv);
                L.w_o = rb(L.w_o);     L.b_o = (const float*)rb(L.b_o);
                L.ln1_g = (const float*)rb(L.ln1_g); L.ln1_b = (const float*)rb(L.ln1_b);
                L.w_1 = rb(L.w_1);     L.b_1 = (const float*)rb(L.b_1);
                L.w_2 = rb(L.w_2);     L.b_2 = (const float*)rb(L.b_2);
                L.ln2_g = (const float*)rb(L.ln2_g); L.ln2_b = (const float*)rb(L.ln2_b);
            }
            HeadW& H = m.head;
            H.E = (const float*)rb(H.E);
            H.v_w = (const float*)rb(H.v_w);   H.b_w = (const float*)rb(H.b_w);
            H.v_mu = (const float*)rb(H.v_mu); H.b_mu = (const float*)rb(H.b_mu);
            H.v_s = (const float*)rb(H.v_s);   H.b_s = (const float*)rb(H.b_s);
            H.v_k1 = (const float*)rb(H.v_k1); H.b_k1 = (const float*)rb(H.b_k1);
            H.v_k2 = (const float*)rb(H.v_k2); H.b_k2 = (const float*)rb(H.b_k2);
        }
    }
    __syncthreads();
    const CallParams& P = *a.P;
    const int s = blockIdx.x * a.wpc + warp;
    if (s >= P.B || a.ss.done[s]) return;  // no block barrier below
    char* wbase = smem + a.w_bytes + (size_t)warp * a.warp_bytes;
    DraftWarp<T, D, F, DH, KVS> dw{m, a, s, lane, a.m.L, a.m.M, a.m.K, a.kv.n_max,
                                   (T*)wbase, nullptr, nullptr};
    const size_t kv_bytes = KVS ? (size_t)a.m.L * 2 * a.kv.n_max * D * sizeof(T) : 0;
    dw.bar = (uint64_t*)(wbase + ((kv_bytes + 15) & ~(size_t)15));
    dw.scratch = (float*)((char*)dw.bar + 16);
    const SeqState& ss = a.ss;
    const int n = ss.n_emit[s], nd = ss.n_draft[s];
    const int M = a.m.M, K = a.m.K, W = 3 * M + K;
    dw.load_kv(nd);
    float x[Regs<D>::n];
    for (int p = nd; p < n; ++p) dw.encode(p, x);
    if (lane == 0) {
        const long long last = n + a.gamma - 2;
        atomicAdd(&a.st->draft_keys, (unsigned long long)((last + 1) * (last + 2) / 2 - (long long)nd * (nd + 1) / 2));
    }
    for (int l = 1; l <= a.gamma; ++l) {
        const int p = n + l - 1;  // index of the drafted event
        float lw[2], mu[2], sg[2], lk[8];
        dw.head(x, lw, mu, sg, lk);
        float* rec = a.heads + ((size_t)s * a.gamma_max + (l - 1)) * W;
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const int o = lane + 32 * r;
            if (o < M) { rec[o] = lw[r]; rec[M + o] = mu[r]; rec[2 * M + o] = sg[r]; }
        }
#pragma unroll
        for (int r = 0; r < 8; ++r) {
            const int o = lane + 32 * r;
            if (o < K) rec[3 * M + o] = lk[r];
        }
        const U4 u = slot_uniforms(P.seed, (uint32_t)s, (uint32_t)p, 0u);
        const int z = wpick<2>(lw, M, u.x, lane);
        const float muz = wget<2>(mu, z), sgz = wget<2>(sg, z);
        const float eps = sqrtf(-2.0f * logf(u.y)) * cospif(2.0f * u.z);
        const float tau = expf(muz + expf(sgz) * eps);
        const int k = wpick<8>(lk, K, u.w, lane);
        const size_t o = (size_t)s * ss.n_max + p;
        if (lane == 0) {
            ss.tau[o] = tau;
            ss.t[o] = ss.t[o - 1] + (double)tau;
            ss.k[o] = k;
        }
        __syncwarp();
        if (l < a.gamma) dw.encode(p, x);
    }
}

// ---------------------------------------------------------------- launcher
template <typename T, int D, int F, int DH>
static cudaError_t launch_t(DraftWArgs& a, int B, int kvs, cudaStream_t st) {
    const int grid = (B + a.wpc - 1) / a.wpc;
    const size_t sm = (size_t)a.w_bytes + (size_t)a.wpc * a.warp_bytes;
    if (kvs) {
        cudaFuncSetAttribute(k_draft_warp<T, D, F, DH, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
        k_draft_warp<T, D, F, DH, true><<<grid, 32 * a.wpc, sm, st>>>(a);
    } else {
        cudaFuncSetAttribute(k_draft_warp<T, D, F, DH, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
        k_draft_warp<T, D, F, DH, false><<<grid, 32 * a.wpc, sm, st>>>(a);
    }
    return cudaGetLastError();
}

int draft_warp_supported(const DevModel& m) {
    if (m.M > 64 || m.K > 256) return 0;
    const int d = m.d, F = m.F, dh = m.dh;
    return (d == 16 && F == 32 && dh == 16) || (d == 32 && F == 128 && dh == 16) ||
           (d == 64 && F == 256 && dh == 16) || (d == 128 && F == 512 && dh == 32);
}

cudaError_t launch_draft_warp(const DevModel& m, const KVCache& kv, const SeqState& ss,
                              const CallParams* dp, int B, int gamma, float* draft_heads,
                              int gamma_max, DevStats* stats, int* err, cudaStream_t st) {
    const size_t SMEM_MAX = 224 * 1024;  // dynamic part; the pointer table is static
    DraftWArgs a{};
    a.m = m; a.kv = kv; a.ss = ss; a.P = dp; a.st = stats; a.heads = draft_heads;
    a.gamma = gamma; a.gamma_max = gamma_max; a.err = err;
    const size_t eb = m.dtype == 1 ? 2 : 4;
    const size_t wb = (m.t.bytes + 15) & ~(size_t)15;
    const size_t scratch = 16 + (size_t)m.d * 4;
    const size_t kvw = ((size_t)m.L * 2 * kv.n_max * m.d * eb + 15) & ~(size_t)15;
    a.w_smem = wb <= 100 * 1024;  // leaves >= 127 KB for resident KV
    a.w_bytes = a.w_smem ? (int)wb : 0;
    const size_t avail = SMEM_MAX - a.w_bytes;
    int kvs = 0, wpc = 4;
    if (kvw + scratch <= avail) {
        kvs = 1;
        wpc = (int)(avail / (kvw + scratch));
        if (wpc > 4) wpc = 4;
        // keep enough CTAs to cover the SMs when the batch is small
        while (wpc > 1 && (B + wpc - 1) / wpc < 120) --wpc;
    }
    a.wpc = wpc;
    a.warp_bytes = (int)(kvs ? kvw + scratch : scratch);
    if (m.dtype == 1) {
        if (m.d == 16) return launch_t<bf16, 16, 32, 16>(a, B, kvs, st);
        if (m.d == 32) return launch_t<bf16, 32, 128, 16>(a, B, kvs, st);
        if (m.d == 64) return launch_t<bf16, 64, 256, 16>(a, B, kvs, st);
        return launch_t<bf16, 128, 512, 32>(a, B, kvs, st);
    }
    if (m.d == 16) return launch_t<float, 16, 32, 16>(a, B, kvs, st);
    if (m.d == 32) return launch_t<float, 32, 128, 16>(a, B, kvs, st);
    if (m.d == 64) return launch_t<float, 64, 256, 16>(a, B, kvs, st);
    return launch_t<float, 128, 512, 32>(a, B, kvs, st);
}

}  // namespace tppsd
