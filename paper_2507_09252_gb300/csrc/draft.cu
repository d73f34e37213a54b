// Draft loop of TPP-SD (Sec. 4.3 "Drafting", Alg. 1): one CTA of 128 threads
// per sequence.
//
// Each round a CTA catches its draft cache up to the last emitted event and
// then drafts gamma events: head of the draft model -> direct sample
// (z ~ Cat(w), eps ~ N(0,1), tau = exp(mu_z + sigma_z eps); k ~ f, Sec. 4.2)
// -> encode the drafted event -> next head.  The critical path of a step is
// a chain of small matrix-vector products; each is spread over the 128
// threads (one thread per output, or input slices reduced through shared
// memory when there are few outputs), and the attention over (head, key
// range) pairs of the four warps.  Weights are read through L1 in an
// [in][out] layout (consecutive threads read consecutive words); the
// sequence's draft KV cache is loaded into shared memory once per round by
// bulk copies and written through to HBM, so all gamma steps read keys on
// chip.
#include <math.h>

#include "common.cuh"
#include "engine.h"
#include "tc_ptx.cuh"

namespace tppsd {

constexpr unsigned FULL = 0xffffffffu;

struct DraftTeamArgs {
    DevModel m;
    KVCache kv;
    SeqState ss;
    const CallParams* P;
    DevStats* st;
    float* heads;  // [Bmax][gamma_max][W]
    int gamma, gamma_max;
    int* err;      // set if the KV bulk load does not complete
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

// y[o] = sum_{i<IN} WT[i][o] xs[i] + b[o] for o < OUT (xs, y in shared
// memory).  Ends with a block barrier.
template <typename TW>
__device__ __forceinline__ void team_mv(const TW* __restrict__ WT, const float* __restrict__ b,
                                        const float* xs, int IN, int OUT, float* y, float* part) {
    const int t = threadIdx.x;
    if (OUT >= 64) {
        for (int o = t; o < OUT; o += 128) {
            float acc = b ? __ldg(b + o) : 0.f;
#pragma unroll 8
            for (int i = 0; i < IN; ++i) acc = fmaf(St<TW>::ld(WT + (size_t)i * OUT + o), xs[i], acc);
            y[o] = acc;
        }
        __syncthreads();
        return;
    }
    // few outputs: G input slices, partial sums reduced through shared memory
    const int OP = OUT <= 32 ? 32 : 64, G = 128 / OP;
    const int o = t % OP, g = t / OP;
    const int per = (IN + G - 1) / G, i0 = g * per, i1 = min(IN, i0 + per);
    float acc = 0.f;
    if (o < OUT) {
#pragma unroll 8
        for (int i = i0; i < i1; ++i) acc = fmaf(St<TW>::ld(WT + (size_t)i * OUT + o), xs[i], acc);
    }
    part[g * OP + o] = acc;
    __syncthreads();
    if (t < OUT) {
        float s = b ? __ldg(b + t) : 0.f;
        for (int gg = 0; gg < G; ++gg) s += part[gg * OP + t];
        y[t] = s;
    }
    __syncthreads();
}

// Attention of one query (qs in shared memory, nh heads of DH) over keys
// 0..n_keys-1 of K/V blocks [nh][stride][DH] (shared or global): warp w
// takes head w % nh and key range w / nh of 4 / nh; lane-strided keys with
// a private online softmax (exp2 units), warp merge by shuffles, then the
// warps of a head merge through shared memory.  Ends with a barrier.
template <typename T, int DH>
__device__ __forceinline__ void team_attend(const float* qs, const T* kb, const T* vb, int stride,
                                            int n_keys, int nh, float* out, float* scratch) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = warp % nh, split = warp / nh, S = 4 / nh;
    const int per = (n_keys + S - 1) / S, lo = split * per, hi = min(n_keys, lo + per);
    const float scale = 1.4426950408889634f / sqrtf((float)DH);
    float q[DH];
#pragma unroll
    for (int c = 0; c < DH; ++c) q[c] = qs[h * DH + c] * scale;
    float mm = -INFINITY, ll = 0.f, o[DH];
#pragma unroll
    for (int c = 0; c < DH; ++c) o[c] = 0.f;
    const T* kh = kb + (size_t)h * stride * DH;
    const T* vh = vb + (size_t)h * stride * DH;
    for (int j = lo + lane; j < hi; j += 32) {
        float kr[DH], vr[DH];
        load_row16<T, DH>(kh + (size_t)j * DH, kr);
        load_row16<T, DH>(vh + (size_t)j * DH, vr);
        float sc = 0.f;
#pragma unroll
        for (int c = 0; c < DH; ++c) sc = fmaf(q[c], kr[c], sc);
        const float mn = fmaxf(mm, sc), corr = exp2f(mm - mn), p = exp2f(sc - mn);
        ll = ll * corr + p;
#pragma unroll
        for (int c = 0; c < DH; ++c) o[c] = fmaf(p, vr[c], o[c] * corr);
        mm = mn;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float m2 = __shfl_xor_sync(FULL, mm, off), l2 = __shfl_xor_sync(FULL, ll, off);
        float a2 = 0.f, b2 = 0.f;
        if (m2 != -INFINITY || mm != -INFINITY) {
            const float mn = fmaxf(mm, m2);
            a2 = mm == -INFINITY ? 0.f : exp2f(mm - mn);
            b2 = m2 == -INFINITY ? 0.f : exp2f(m2 - mn);
            mm = mn;
        }
        ll = ll * a2 + l2 * b2;
#pragma unroll
        for (int c = 0; c < DH; ++c) o[c] = o[c] * a2 + __shfl_xor_sync(FULL, o[c], off) * b2;
    }
    float* sw = scratch + warp * (DH + 2);
    if (lane == 0) {
        sw[0] = mm;
        sw[1] = ll;
#pragma unroll
        for (int c = 0; c < DH; ++c) sw[2 + c] = o[c];
    }
    __syncthreads();
    for (int t = threadIdx.x; t < nh * DH; t += 128) {
        const int hh = t / DH, c = t % DH;
        float M = -INFINITY;
        for (int sp = 0; sp < S; ++sp) M = fmaxf(M, scratch[(sp * nh + hh) * (DH + 2)]);
        float L = 0.f, O = 0.f;
        for (int sp = 0; sp < S; ++sp) {
            const float* src = scratch + (sp * nh + hh) * (DH + 2);
            if (src[0] == -INFINITY) continue;
            const float e = exp2f(src[0] - M);
            L += src[1] * e;
            O += src[2 + c] * e;
        }
        out[t] = O / L;
    }
    __syncthreads();
}

// Residual add + LayerNorm of x (shared, d) by warp 0; also its rounded copy.
template <typename T>
__device__ __forceinline__ void team_add_ln(float* x, const float* y, float* xin, int d, const float* g,
                                            const float* b) {
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        float sum = 0.f;
        for (int i = lane; i < d; i += 32) { x[i] += y[i]; sum += x[i]; }
        const float mean = warp_sum(sum) / d;
        float var = 0.f;
        for (int i = lane; i < d; i += 32) var += (x[i] - mean) * (x[i] - mean);
        const float inv = 1.0f / sqrtf(warp_sum(var) / d + LN_EPS);
        for (int i = lane; i < d; i += 32) {
            const float v = (x[i] - mean) * inv * g[i] + b[i];
            x[i] = v;
            xin[i] = St<T>::rnd(v);
        }
    }
    __syncthreads();
}

template <typename T, int DH, bool KVS>
__global__ void __launch_bounds__(128) k_draft_team(DraftTeamArgs a) {
    extern __shared__ __align__(16) char smem[];
    const int s = blockIdx.x;
    const CallParams& P = *a.P;
    if (s >= P.B || a.ss.done[s]) return;
    const int tid = threadIdx.x;
    const DevModelT& m = a.m.t;
    const int d = a.m.d, F = a.m.F, M = a.m.M, K = a.m.K, W = 3 * M + K, L = a.m.L, NH = d / DH;
    const int n_max = a.kv.n_max;
    // shared layout: [resident KV][mbarrier][work vectors]
    const size_t kvb = KVS ? (((size_t)L * 2 * n_max * d * sizeof(T) + 15) & ~(size_t)15) : 0;
    T* kvs = (T*)smem;
    uint64_t* bar = (uint64_t*)(smem + kvb);
    float* x = (float*)(smem + kvb + 16);
    float* xin = x + d;
    float* qkv = xin + d;
    float* att = qkv + 3 * d;
    float* hid = att + d;
    float* e = hid + F;
    float* av = e + 3 * d;
    float* hd = av + d;
    float* part = hd + ((W + 3) & ~3);
    float* attn = part + 128;
    const SeqState& ss = a.ss;
    const int n = ss.n_emit[s], nd = ss.n_draft[s];
    auto gk = [&](int l, int w) -> T* {
        return (T*)(w ? a.kv.v : a.kv.k) + (((size_t)l * a.kv.Bmax + s) * NH) * (size_t)n_max * DH;
    };
    auto sk = [&](int l, int w) -> T* { return kvs + (((size_t)l * 2 + w) * NH) * (size_t)n_max * DH; };
    if (KVS && nd > 0) {
        // each (layer, K/V, head) block of positions 0..nd-1 is contiguous in HBM
        if (tid == 0) {
            const uint32_t bytes = (uint32_t)nd * DH * sizeof(T);
            mbar_init(bar, 1);
            mbar_fence_init();
            mbar_arrive_expect_tx(bar, bytes * (uint32_t)(L * 2 * NH));
            for (int l = 0; l < L; ++l)
                for (int w = 0; w < 2; ++w)
                    for (int h = 0; h < NH; ++h)
                        bulk_load(sk(l, w) + (size_t)h * n_max * DH, gk(l, w) + (size_t)h * n_max * DH, bytes, bar);
        }
        __syncthreads();
        mbar_wait(bar, 0, a.err, 12);
    }
    auto encode = [&](int p) {
        const size_t so = (size_t)s * ss.n_max + p;
        const double t = ss.t[so];
        const int k = min(max(ss.k[so], 0), K - 1);
        for (int i = tid; i < d; i += 128) {
            const double ang = t * m.omega[i >> 1];
            const double red = fma(-6.283185307179586476925, rint(ang * 0.15915494309189533577), ang);
            float sv, cv;
            sincosf((float)red, &sv, &cv);
            const float v = ((i & 1) ? cv : sv) + m.type_emb[(size_t)k * d + i];
            x[i] = v;
            xin[i] = St<T>::rnd(v);
        }
        __syncthreads();
        for (int l = 0; l < L; ++l) {
            const LayerW& Wl = m.layer[l];
            team_mv<T>((const T*)Wl.w_qkv, Wl.b_qkv, xin, d, 3 * d, qkv, part);
            for (int i = tid; i < 3 * d; i += 128) {
                const float v = St<T>::rnd(qkv[i]);
                qkv[i] = v;
                if (i >= d) {
                    const int w = i < 2 * d ? 0 : 1, c = i - d - w * d, hh = c / DH, ee = c - hh * DH;
                    const size_t off = ((size_t)hh * n_max + p) * DH + ee;
                    St<T>::st(gk(l, w) + off, v);
                    if (KVS) St<T>::st(sk(l, w) + off, v);
                }
            }
            __syncthreads();
            const T* kb = KVS ? sk(l, 0) : gk(l, 0);
            const T* vb = KVS ? sk(l, 1) : gk(l, 1);
            team_attend<T, DH>(qkv, kb, vb, n_max, p + 1, NH, att, attn);
            for (int i = tid; i < d; i += 128) att[i] = St<T>::rnd(att[i]);
            __syncthreads();
            team_mv<T>((const T*)Wl.w_o, Wl.b_o, att, d, d, e, part);
            team_add_ln<T>(x, e, xin, d, Wl.ln1_g, Wl.ln1_b);
            team_mv<T>((const T*)Wl.w_1, Wl.b_1, xin, d, F, hid, part);
            for (int i = tid; i < F; i += 128) hid[i] = St<T>::rnd(fmaxf(hid[i], 0.f));
            __syncthreads();
            team_mv<T>((const T*)Wl.w_2, Wl.b_2, hid, F, d, e, part);
            team_add_ln<T>(x, e, xin, d, Wl.ln2_g, Wl.ln2_b);
        }
    };
    for (int p = nd; p < n; ++p) encode(p);
    if (tid == 0) {
        const long long last = n + a.gamma - 2;  // last position the round encodes
        atomicAdd(&a.st->draft_keys, (unsigned long long)((last + 1) * (last + 2) / 2 - (long long)nd * (nd + 1) / 2));
    }
    const HeadW& H = m.head;
    for (int l = 1; l <= a.gamma; ++l) {
        const int p = n + l - 1;  // index of the drafted event
        // head (Sec. 4.2): e = E h, a = tanh(V_k1 h + b), then the small maps
        team_mv<float>(H.E, nullptr, x, d, 3 * d, e, part);
        team_mv<float>(H.v_k1, H.b_k1, x, d, d, av, part);
        for (int i = tid; i < d; i += 128) av[i] = tanhf(av[i]);
        __syncthreads();
        team_mv<float>(H.v_w, H.b_w, e, d, M, hd, part);
        team_mv<float>(H.v_mu, H.b_mu, e + d, d, M, hd + M, part);
        team_mv<float>(H.v_s, H.b_s, e + 2 * d, d, M, hd + 2 * M, part);
        team_mv<float>(H.v_k2, H.b_k2, av, d, K, hd + 3 * M, part);
        const int warp = tid >> 5;
        if (warp < 2) {  // log-softmax of w (warp 0) and f (warp 1)
            float* v = warp == 0 ? hd : hd + 3 * M;
            const int nn = warp == 0 ? M : K, lane = tid & 31;
            float mx = -INFINITY;
            for (int i = lane; i < nn; i += 32) mx = fmaxf(mx, v[i]);
            mx = warp_max(mx);
            float sm = 0.f;
            for (int i = lane; i < nn; i += 32) sm += expf(v[i] - mx);
            const float lz = mx + logf(warp_sum(sm));
            __syncwarp();
            for (int i = lane; i < nn; i += 32) v[i] -= lz;
        }
        __syncthreads();
        float* rec = a.heads + ((size_t)s * a.gamma_max + (l - 1)) * W;
        for (int i = tid; i < W; i += 128) rec[i] = hd[i];
        if (tid == 0) {
            const U4 u = slot_uniforms(P.seed, (uint32_t)s, (uint32_t)p, 0u);
            const float tau = draw_tau(hd, M, u.x, u.y, u.z);
            const int k = pick_categorical_log(hd + 3 * M, K, u.w);
            const size_t o = (size_t)s * ss.n_max + p;
            ss.tau[o] = tau;
            ss.t[o] = ss.t[o - 1] + (double)tau;
            ss.k[o] = k;
        }
        __syncthreads();
        if (l < a.gamma) encode(p);
    }
}

template <typename T, int DH>
static cudaError_t launch_team(DraftTeamArgs& a, int B, int kvs, size_t sm, cudaStream_t st) {
    if (kvs) {
        cudaFuncSetAttribute(k_draft_team<T, DH, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
        k_draft_team<T, DH, true><<<B, 128, sm, st>>>(a);
    } else {
        cudaFuncSetAttribute(k_draft_team<T, DH, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
        k_draft_team<T, DH, false><<<B, 128, sm, st>>>(a);
    }
    return cudaGetLastError();
}

int draft_team_supported(const DevModel& m) {
    const int nh = m.nh;
    if (!(nh == 1 || nh == 2 || nh == 4) || !(m.dh == 16 || m.dh == 32)) return 0;
    return m.M <= 64 && m.K <= 256;
}

// The sequence's draft KV is kept in shared memory for the round when that
// still leaves room for two CTAs per SM; otherwise it is read from HBM/L2.
cudaError_t launch_draft_team(const DevModel& m, const KVCache& kv, const SeqState& ss,
                              const CallParams* dp, int B, int gamma, float* draft_heads,
                              int gamma_max, DevStats* stats, int* err, cudaStream_t st) {
    DraftTeamArgs a{};
    a.m = m; a.kv = kv; a.ss = ss; a.P = dp; a.st = stats; a.heads = draft_heads;
    a.gamma = gamma; a.gamma_max = gamma_max; a.err = err;
    const size_t eb = m.dtype == 1 ? 2 : 4;
    const int W = 3 * m.M + m.K;
    const size_t fl = sizeof(float) * (10 * (size_t)m.d + m.F + ((W + 3) & ~3) + 128 + 4 * 66) + 16;
    const size_t kvb = ((size_t)m.L * 2 * kv.n_max * m.d * eb + 15) & ~(size_t)15;
    const int kvs = kvb + fl <= 110 * 1024;
    const size_t sm = (kvs ? kvb : 0) + fl;
    if (m.dtype == 0) {
        if (m.dh == 16) return launch_team<float, 16>(a, B, kvs, sm, st);
        return launch_team<float, 32>(a, B, kvs, sm, st);
    }
    if (m.dh == 16) return launch_team<bf16, 16>(a, B, kvs, sm, st);
    return launch_team<bf16, 32>(a, B, kvs, sm, st);
}

}  // namespace tppsd
