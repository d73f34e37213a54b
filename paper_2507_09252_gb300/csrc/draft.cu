// Draft loop of TPP-SD (Sec. 4.3 "Drafting", Alg. 1): one CTA of 128 threads
// per sequence.
//
// Each round a CTA catches its draft cache up to the last emitted event and
// then drafts gamma events: head of the draft model -> direct sample
// (z ~ Cat(w), eps ~ N(0,1), tau = exp(mu_z + sigma_z eps); k ~ f, Sec. 4.2)
// -> encode the drafted event -> next head.  The critical path is a chain
// of small matrix-vector products, each spread over the 128 threads: one
// thread per output when there are many outputs, otherwise input slices
// whose partial sums are reduced through shared memory, with the bias,
// residual add and LayerNorm folded into that reduction (d <= 32).  The
// attention runs over (head, key range) pairs of the four warps.  The two
// components of the sample (time by warp 0, mark by warp 1) are drawn in
// parallel with warp scans.  Weights are read through L1 in an [in][out]
// layout (consecutive threads read consecutive words); the sequence's draft
// KV cache is loaded into shared memory once per round by bulk copies and
// written through to HBM, so all gamma steps read keys on chip.
#include <math.h>

#include <algorithm>
#include <stdlib.h>

#include "common.cuh"
#include "engine.h"
#include "tc_ptx.cuh"

namespace tppsd {

constexpr unsigned FULL = 0xffffffffu;

// Barrier of the NT threads that work on one sequence: 128-thread teams use
// named barrier 1 or 2 (a CTA holds one or two such teams), a 256-thread
// team named barrier 1.
template <int NT = 128>
__device__ __forceinline__ void team_sync() {
    if constexpr (NT == 256) {
        asm volatile("bar.sync 1, 256;" ::: "memory");
    } else {
        if (threadIdx.x < 128) asm volatile("bar.sync 1, 128;" ::: "memory");
        else asm volatile("bar.sync 2, 128;" ::: "memory");
    }
}

struct DraftTeamArgs {
    DevModel m;
    KVCache kv;
    SeqState ss;
    const CallParams* P;
    DevStats* st;
    float* heads;  // [Bmax][gamma_max][W]
    int gamma, gamma_max;
    int* err;      // set if a bulk copy of KV or weights does not complete
    int ring_nst, ring_ch;  // streamed KV (k_draft_team without resident KV): stages, keys per stage
    DraftEmbed emb;         // lane form: the target's verify rows (emb.x null: not written here)
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

// sum_{i<i1} WT[i][o] xs[i] over i from i0, with four independent partial
// sums (WT is [IN][OUT], xs in shared memory).
template <typename TW>
__device__ __forceinline__ float dot_range(const TW* __restrict__ WT, int OUT, int o, const float* xs, int i0,
                                           int i1) {
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
    const TW* w = WT + (size_t)i0 * OUT + o;
    int i = i0;
#pragma unroll 2
    for (; i + 4 <= i1; i += 4, w += 4 * (size_t)OUT) {
        a0 = fmaf(St<TW>::ld(w), xs[i], a0);
        a1 = fmaf(St<TW>::ld(w + OUT), xs[i + 1], a1);
        a2 = fmaf(St<TW>::ld(w + 2 * (size_t)OUT), xs[i + 2], a2);
        a3 = fmaf(St<TW>::ld(w + 3 * (size_t)OUT), xs[i + 3], a3);
    }
    for (; i < i1; ++i, w += OUT) a0 = fmaf(St<TW>::ld(w), xs[i], a0);
    return (a0 + a1) + (a2 + a3);
}

// Floats of the partial-sum buffer of team_gemv for a model of width d and
// FFN width F and a team of NT threads: G * OUT <= max(NT * 8, OUT) for
// every product of the step.
__host__ __device__ inline int team_gp_floats(int d, int F, int NT = 128) {
    int g = 8 * NT;
    if (4 * d > g) g = 4 * d;
    if (F > g) g = F;
    return g;
}

// acc[v] += sum_{i0 <= i < i1} W[i][v] in[i] for the 16 bytes of weights of
// row i at col (row stride OUT elements): eight 16-byte loads in flight.
template <typename TW>
__device__ __forceinline__ void gemv_slice(const TW* __restrict__ col, int OUT, const float* in, int i0, int i1,
                                           float (&acc)[16 / sizeof(TW)]) {
    constexpr int V = 16 / sizeof(TW), U = 8;
    auto fma_row = [&](const uint4& w, float xv) {
        if constexpr (sizeof(TW) == 2) {
            const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&w);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float2 f = __bfloat1622float2(h[j]);
                acc[2 * j] = fmaf(f.x, xv, acc[2 * j]);
                acc[2 * j + 1] = fmaf(f.y, xv, acc[2 * j + 1]);
            }
        } else {
            acc[0] = fmaf(__uint_as_float(w.x), xv, acc[0]);
            acc[1] = fmaf(__uint_as_float(w.y), xv, acc[1]);
            acc[2] = fmaf(__uint_as_float(w.z), xv, acc[2]);
            acc[3] = fmaf(__uint_as_float(w.w), xv, acc[3]);
        }
    };
    static_assert(V == 8 || V == 4, "16-byte rows of 8 bf16 or 4 fp32 weights");
    const TW* p = col + (size_t)i0 * OUT;
    int i = i0;
    for (; i + U <= i1; i += U, p += (size_t)U * OUT) {
        uint4 w[U];
#pragma unroll
        for (int u = 0; u < U; ++u) w[u] = *reinterpret_cast<const uint4*>(p + (size_t)u * OUT);
#pragma unroll
        for (int u = 0; u < U; ++u) fma_row(w[u], in[i + u]);
    }
    for (; i < i1; ++i, p += OUT) fma_row(*reinterpret_cast<const uint4*>(p), in[i]);
}

// Partial sums of the product [W1 | W2]^T in (W1 [IN][OUT1], W2 [IN][OUT2],
// [in][out] layout, OUT1 and OUT2 multiples of V = 16 bytes / weight):
// thread t takes the V consecutive outputs of column group t % NC over input
// slice t / NC of G (NC = (OUT1 + OUT2) / V groups; G = 128 / NC, but no
// slice under 8 inputs; all groups per thread, G = 1, once NC >= 128).
// part[g * OUT + o] receives slice g's sum of output o (OUT = OUT1 + OUT2).
// Returns G; ends with a team barrier.
template <typename TW, int NT = 128>
__device__ __forceinline__ int team_gemv(const TW* __restrict__ W1, int OUT1, const TW* __restrict__ W2, int OUT2,
                                         const float* in, int IN, float* part) {
    constexpr int V = 16 / sizeof(TW);
    const int t = threadIdx.x & (NT - 1), OUT = OUT1 + OUT2, NC = OUT / V;
    const int G = NC >= NT ? 1 : max(1, min(NT / NC, IN / 8));
    const int per = (IN + G - 1) / G;
    for (int c = t; c < NC * G; c += NT) {
        const int cg = c % NC, g = c / NC, o = cg * V;
        const int i0 = g * per, i1 = min(IN, i0 + per);
        float acc[V];
#pragma unroll
        for (int v = 0; v < V; ++v) acc[v] = 0.f;
        if (o < OUT1) gemv_slice<TW>(W1 + o, OUT1, in, i0, i1, acc);
        else gemv_slice<TW>(W2 + (o - OUT1), OUT2, in, i0, i1, acc);
        float4* dst = reinterpret_cast<float4*>(part + (size_t)g * OUT + o);
#pragma unroll
        for (int v = 0; v < V; v += 4) dst[v / 4] = make_float4(acc[v], acc[v + 1], acc[v + 2], acc[v + 3]);
    }
    team_sync<NT>();
    return G;
}

// Output o of a team_gemv: slice sums in slice order.
__device__ __forceinline__ float gemv_out(const float* part, int OUT, int G, int o) {
    float v = part[o];
    for (int g = 1; g < G; ++g) v += part[(size_t)g * OUT + o];
    return v;
}

// Residual add + LayerNorm of d <= 32 values by warp 0 (lane j < d holds
// the summed output j): x = LN(x + y), xin its rounded copy.
template <typename T>
__device__ __forceinline__ void warp_resid_ln(float yv, float* x, float* xin, int d, const float* g,
                                              const float* b) {
    const int lane = threadIdx.x & 31;
    const bool live = lane < d;
    const float v = live ? x[lane] + yv : 0.f;
    const float mean = warp_sum(v) / d;
    const float c = live ? v - mean : 0.f;
    const float inv = 1.0f / sqrtf(warp_sum(c * c) / d + LN_EPS);
    if (live) {
        const float o = c * inv * g[lane] + b[lane];
        x[lane] = o;
        xin[lane] = St<T>::rnd(o);
    }
}

// Online-softmax state of one lane over the keys it has seen (exp2 units).
template <int DH>
struct AttState {
    float q[DH], o[DH], mm, ll;
    __device__ __forceinline__ void init(const float* qs, int h) {
        const float scale = 1.4426950408889634f / sqrtf((float)DH);
#pragma unroll
        for (int c = 0; c < DH; ++c) {
            q[c] = qs[h * DH + c] * scale;
            o[c] = 0.f;
        }
        mm = -INFINITY;
        ll = 0.f;
    }
    // one key: K row kr, V row at vp
    template <typename T>
    __device__ __forceinline__ void add(const T* kp, const T* vp) {
        float kr[DH], vr[DH];
        load_row16<T, DH>(kp, kr);
        load_row16<T, DH>(vp, vr);
        float sc = 0.f;
#pragma unroll
        for (int c = 0; c < DH; ++c) sc = fmaf(q[c], kr[c], sc);
        const float mn = fmaxf(mm, sc), corr = exp2f(mm - mn), p = exp2f(sc - mn);
        ll = ll * corr + p;
#pragma unroll
        for (int c = 0; c < DH; ++c) o[c] = fmaf(p, vr[c], o[c] * corr);
        mm = mn;
    }
};

// Merge of the lanes' states (shuffles), then of the warps of a head
// (shared memory), into out[nh * DH].  Softmax: the output is rounded to
// the storage type.  attnhp (App. D.4): the normaliser is 1 + sum_j f_j (an
// extra term exp(0)) and the fp32 output is kept.  Ends with a barrier.
template <typename T, int DH, int NT = 128>
__device__ __forceinline__ void team_attend_merge(AttState<DH>& a, int nh, float* out, float* scratch,
                                                  bool attnhp) {
    const int warp = (threadIdx.x & (NT - 1)) >> 5, lane = threadIdx.x & 31, S = NT / 32 / nh;
    float mm = a.mm, ll = a.ll;
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
        for (int c = 0; c < DH; ++c) a.o[c] = a.o[c] * a2 + __shfl_xor_sync(FULL, a.o[c], off) * b2;
    }
    float* sw = scratch + warp * (DH + 2);
    if (lane == 0) {
        sw[0] = mm;
        sw[1] = ll;
#pragma unroll
        for (int c = 0; c < DH; ++c) sw[2 + c] = a.o[c];
    }
    team_sync<NT>();
    for (int t = threadIdx.x & (NT - 1); t < nh * DH; t += NT) {
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
        out[t] = attnhp ? O / (L + exp2f(-M)) : St<T>::rnd(O / L);
    }
    team_sync<NT>();
}

// Attention of one query (qs in shared memory, nh heads of DH) over keys
// 0..n_keys-1 of K/V blocks [nh][stride][DH] in shared memory: warp w takes
// head w % nh and key range w / nh of 4 / nh; lane-strided keys with a
// private online softmax, then team_attend_merge.  Ends with a barrier.
template <typename T, int DH, int NT = 128>
__device__ __forceinline__ void team_attend(const float* qs, const T* kb, const T* vb, int stride,
                                            int n_keys, int nh, float* out, float* scratch,
                                            bool attnhp = false) {
    const int warp = (threadIdx.x & (NT - 1)) >> 5, lane = threadIdx.x & 31;
    const int h = warp % nh, split = warp / nh, S = NT / 32 / nh;
    const int per = (n_keys + S - 1) / S, lo = split * per, hi = min(n_keys, lo + per);
    AttState<DH> a;
    a.init(qs, h);
    const T* kh = kb + (size_t)h * stride * DH;
    const T* vh = vb + (size_t)h * stride * DH;
    for (int j = lo + lane; j < hi; j += 32) a.template add<T>(kh + (size_t)j * DH, vh + (size_t)j * DH);
    team_attend_merge<T, DH, NT>(a, nh, out, scratch, attnhp);
}

// Ring of shared-memory stages through which team_attend_stream streams a
// sequence's K/V from HBM: stage i holds ch keys of every head, K then V
// per head ([nh][2][ch][DH]); full[i] completes when its bulk copies land.
struct KvRing {
    char* buf;
    uint64_t* full;
    int nst, ch;
    uint32_t used;  // chunks consumed so far (the same in every thread)
    bool ok;        // false after a wait gave up: no further copies or waits
};

// team_attend over keys 0..n_keys-1 of HBM blocks [nh][stride][DH] (the
// draft KV cache of one layer and sequence): thread 0 keeps nst chunks of ch
// keys in flight by bulk copies (all heads, K and V), the team consumes them
// in order, and a team barrier after each chunk frees its stage for the
// chunk nst ahead.  Keys written by this CTA's generic stores must be fenced
// (fence_proxy_async_global) before the barrier that precedes the call.
// Ends with a barrier.
template <typename T, int DH, int NT = 128>
__device__ __forceinline__ void team_attend_stream(const float* qs, const T* kg, const T* vg, int stride, int n_keys,
                                                int nh, float* out, float* scratch, KvRing& r, int* err,
                                                bool attnhp = false) {
    const int tid = threadIdx.x & (NT - 1), warp = tid >> 5, lane = tid & 31;
    const int h = warp % nh, split = warp / nh, S = NT / 32 / nh;
    const int nch = (n_keys + r.ch - 1) / r.ch;
    const size_t hs = (size_t)r.ch * DH, ss = 2 * (size_t)nh * hs;
    auto issue = [&](int c) {
        const uint32_t u = r.used + (uint32_t)c;
        const int st = (int)(u % (uint32_t)r.nst);
        const int k0 = c * r.ch, cnt = min(r.ch, n_keys - k0);
        const uint32_t bytes = (uint32_t)cnt * DH * sizeof(T);
        T* dst = (T*)r.buf + st * ss;
        mbar_arrive_expect_tx(r.full + st, 2u * nh * bytes);
        for (int hh = 0; hh < nh; ++hh) {
            const size_t src = ((size_t)hh * stride + k0) * DH;
            bulk_load(dst + (2 * hh) * hs, kg + src, bytes, r.full + st);
            bulk_load(dst + (2 * hh + 1) * hs, vg + src, bytes, r.full + st);
        }
    };
    if (tid == 0 && r.ok) {
        fence_proxy_async_global();
        for (int c = 0; c < min(r.nst, nch); ++c) issue(c);
    }
    AttState<DH> a;
    a.init(qs, h);
    for (int c = 0; c < nch; ++c) {
        const uint32_t u = r.used + (uint32_t)c;
        const int st = (int)(u % (uint32_t)r.nst);
        if (r.ok) r.ok = mbar_wait(r.full + st, (u / (uint32_t)r.nst) & 1u, err, 15);
        const int cnt = min(r.ch, n_keys - c * r.ch);
        const int per = (cnt + S - 1) / S, lo = split * per, hi = min(cnt, lo + per);
        const T* kh = (const T*)r.buf + st * ss + (2 * h) * hs;
        for (int j = lo + lane; j < hi; j += 32) a.template add<T>(kh + (size_t)j * DH, kh + hs + (size_t)j * DH);
        team_sync<NT>();
        if (tid == 0 && r.ok && c + r.nst < nch) issue(c + r.nst);
    }
    r.used += (uint32_t)nch;
    team_attend_merge<T, DH, NT>(a, nh, out, scratch, attnhp);
}

// Warp-parallel log-softmax of n <= 32*R values v[] (shared) in place, then
// the smallest index whose running sum of probabilities reaches u * total.
template <int R>
__device__ __forceinline__ int warp_logsoftmax_pick(float* v, int n, float u) {
    const int lane = threadIdx.x & 31;
    float x[R];
    float mx = -INFINITY;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int i = lane + 32 * r;
        x[r] = i < n ? v[i] : -INFINITY;
        mx = fmaxf(mx, x[r]);
    }
    mx = warp_max(mx);
    float sm = 0.f;
#pragma unroll
    for (int r = 0; r < R; ++r) sm += lane + 32 * r < n ? expf(x[r] - mx) : 0.f;
    const float lz = mx + logf(warp_sum(sm));
    float p[R], tot = 0.f;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int i = lane + 32 * r;
        p[r] = 0.f;
        if (i < n) {
            x[r] -= lz;
            v[i] = x[r];
            p[r] = expf(x[r]);
        }
        tot += p[r];
    }
    const float target = u * warp_sum(tot);
    float base = 0.f;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        float c = p[r];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const float t = __shfl_up_sync(FULL, c, o);
            if (lane >= o) c += t;
        }
        const unsigned hit = __ballot_sync(FULL, lane + 32 * r < n && base + c >= target);
        if (hit) return 32 * r + __ffs(hit) - 1;
        base += __shfl_sync(FULL, c, 31);
    }
    return n - 1;
}

// Copy of the transposed model's pointer table whose pointers are rebased
// onto a staged copy of its bytes at dst.
__device__ void rebase_model(DevModelT& m, const DevModelT& src, int L, const char* dst) {
    m = src;
    auto rb = [&](const void* p) { return p ? dst + ((const char*)p - src.base) : nullptr; };
    m.type_emb = (const float*)rb(m.type_emb);
    m.tenc = (const double*)rb(m.tenc);
    for (int l = 0; l < L; ++l) {
        LayerW& w = m.layer[l];
        w.w_qkv = rb(w.w_qkv); w.b_qkv = (const float*)rb(w.b_qkv);
        w.w_o = rb(w.w_o);     w.b_o = (const float*)rb(w.b_o);
        w.ln1_g = (const float*)rb(w.ln1_g); w.ln1_b = (const float*)rb(w.ln1_b);
        w.w_1 = rb(w.w_1);     w.b_1 = (const float*)rb(w.b_1);
        w.w_2 = rb(w.w_2);     w.b_2 = (const float*)rb(w.b_2);
        w.ln2_g = (const float*)rb(w.ln2_g); w.ln2_b = (const float*)rb(w.ln2_b);
    }
    HeadW& h = m.head;
    h.E = (const float*)rb(h.E);
    h.v_w = (const float*)rb(h.v_w);   h.b_w = (const float*)rb(h.b_w);
    h.v_mu = (const float*)rb(h.v_mu); h.b_mu = (const float*)rb(h.b_mu);
    h.v_s = (const float*)rb(h.v_s);   h.b_s = (const float*)rb(h.b_s);
    h.v_k1 = (const float*)rb(h.v_k1); h.b_k1 = (const float*)rb(h.b_k1);
    h.v_k2 = (const float*)rb(h.v_k2); h.b_k2 = (const float*)rb(h.b_k2);
    m.base = dst;
}

// TEAMS sequences per CTA, NT threads each (128, or 256 when there are
// fewer sequences than SMs, so that each sequence's chain of products and
// key ranges is split twice as finely).  With WS the draft model is staged
// once per CTA in shared memory (shared by its two 128-thread teams), so no
// weight read leaves the SM; otherwise weights are read through L1.
template <typename T, int DH, bool KVS, bool WS, int NT>
__global__ void __launch_bounds__(WS ? 256 : NT) k_draft_team(DraftTeamArgs a, int area_bytes) {
    static_assert(!WS || NT == 128, "two teams of 128 share a staged model");
    constexpr int TEAMS = WS ? 2 : 1;
    pdl_wait();
    extern __shared__ __align__(16) char smem[];
    __shared__ double t_new_s[TEAMS];
    __shared__ int k_new_s[TEAMS];
    __shared__ DevModelT msh;
    __shared__ uint64_t wbar;
    const int team = threadIdx.x / NT;
    const int s = blockIdx.x * TEAMS + team;
    const CallParams& P = *a.P;
    char* area = smem;
    if (WS) {
        const uint32_t wb = (uint32_t)a.m.t.bytes;
        if (threadIdx.x == 0) {
            mbar_init(&wbar, 1);
            mbar_fence_init();
            mbar_arrive_expect_tx(&wbar, wb);
            bulk_load(smem, a.m.t.base, wb, &wbar);
            rebase_model(msh, a.m.t, a.m.L, smem);
        }
        __syncthreads();
        mbar_wait(&wbar, 0, a.err, 13);
        area = smem + wb + (size_t)team * area_bytes;
    }
    if (s >= P.B || a.ss.done[s]) return;  // the rest synchronises within the team only
    double& t_new = t_new_s[team];
    int& k_new = k_new_s[team];
    const int tid = threadIdx.x & (NT - 1), warp = tid >> 5, lane = tid & 31;
    const DevModelT& m = WS ? msh : a.m.t;
    const int d = a.m.d, F = a.m.F, M = a.m.M, K = a.m.K, W = 3 * M + K, L = a.m.L, NH = d / DH;
    const int n_max = a.kv.n_max;
    // team area: [resident KV][8 mbarriers][KV ring (streamed KV)][work vectors]
    const size_t kvb = KVS ? (((size_t)L * 2 * n_max * d * sizeof(T) + 15) & ~(size_t)15) : 0;
    const size_t ringb = KVS ? 0 : (size_t)a.ring_nst * a.ring_ch * 2 * d * sizeof(T);
    T* kvs = (T*)area;
    uint64_t* bar = (uint64_t*)(area + kvb);
    KvRing ring{area + kvb + 64, bar + 1, a.ring_nst, a.ring_ch, 0u, true};
    if (!KVS) {
        if (tid == 0) {
            for (int i = 0; i < ring.nst; ++i) mbar_init(ring.full + i, 1);
            mbar_fence_init();
        }
        team_sync<NT>();
    }
    float* x = (float*)(area + kvb + 64 + ringb);
    float* zin = x + d;   // rounded temporal encoding; [zin | xin] is the AttNHP QKV input
    float* xin = zin + d;
    float* qkv = xin + d;
    float* att = qkv + 3 * d;
    float* hid = att + d;
    float* y = hid + F;
    float* e = y + d;  // E h (3d) | tanh(V_k1 h + b_k1) (d)
    float* hd = e + 4 * d;
    float* part = hd + ((W + 3) & ~3);  // team_gemv partial sums (16-byte aligned)
    float* attn = part + team_gp_floats(d, F, NT);
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
        team_sync<NT>();
        mbar_wait(bar, 0, a.err, 12);
    }
    // x = LN(x + W_T in + b): the product, then the residual add and
    // LayerNorm (by warp 0, in registers when d <= 32).  Ends synced.
    auto proj_resid_ln = [&](const T* WT, const float* bias, const float* in, int IN, const float* g,
                             const float* b) {
        const int G = team_gemv<T, NT>(WT, d, nullptr, 0, in, IN, part);
        if (d <= 32) {
            if (warp == 0) {
                const float v = lane < d ? bias[lane] + gemv_out(part, d, G, lane) : 0.f;
                warp_resid_ln<T>(v, x, xin, d, g, b);
            }
            team_sync<NT>();
            return;
        }
        if (warp == 0) {
            float sum = 0.f;
            for (int i = lane; i < d; i += 32) {
                x[i] += bias[i] + gemv_out(part, d, G, i);
                sum += x[i];
            }
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
        team_sync<NT>();
    };
    // Q, K, V of position p from the QKV input qin (IN wide); K and V
    // appended to the cache (and its resident copy).  Ends synced.
    auto qkv_step = [&](const LayerW& Wl, int l, int p, const float* qin, int IN) {
        const int G = team_gemv<T, NT>((const T*)Wl.w_qkv, 3 * d, nullptr, 0, qin, IN, part);
        for (int o = tid; o < 3 * d; o += NT) {
            const float v = St<T>::rnd(Wl.b_qkv[o] + gemv_out(part, 3 * d, G, o));
            qkv[o] = v;
            if (o >= d) {
                const int w = o < 2 * d ? 0 : 1, c = o - d - w * d, hh = c / DH, ee = c - hh * DH;
                const size_t off = ((size_t)hh * n_max + p) * DH + ee;
                St<T>::st(gk(l, w) + off, v);
                if (KVS) St<T>::st(sk(l, w) + off, v);
            }
        }
        if (!KVS) fence_proxy_async_global();  // the streamed attention reads them back by bulk copy
        team_sync<NT>();
    };
    auto attend = [&](int l, int p, bool attnhp) {
        if (KVS) team_attend<T, DH, NT>(qkv, sk(l, 0), sk(l, 1), n_max, p + 1, NH, att, attn, attnhp);
        else team_attend_stream<T, DH, NT>(qkv, gk(l, 0), gk(l, 1), n_max, p + 1, NH, att, attn, ring, a.err, attnhp);
    };
    // Layers of the encode step at position p from x / xin (set and synced
    // by the caller); leaves the final hidden state in x (synced).
    const bool att_enc = a.m.enc == 2;
    auto layers = [&](int p) {
        if (att_enc) {
            // AttNHP (App. D.4): q, k, v = W [z; h] + b, a = sum f v / (1 + sum f),
            // h <- h + tanh(a)
            for (int l = 0; l < L; ++l) {
                qkv_step(m.layer[l], l, p, zin, 2 * d);
                attend(l, p, true);
                for (int i = tid; i < d; i += NT) {
                    x[i] += tanhf(att[i]);
                    xin[i] = St<T>::rnd(x[i]);
                }
                team_sync<NT>();
            }
            return;
        }
        for (int l = 0; l < L; ++l) {
            const LayerW& Wl = m.layer[l];
            qkv_step(Wl, l, p, xin, d);
            attend(l, p, false);
            proj_resid_ln((const T*)Wl.w_o, Wl.b_o, att, d, Wl.ln1_g, Wl.ln1_b);
            {
                const int G = team_gemv<T, NT>((const T*)Wl.w_1, F, nullptr, 0, xin, d, part);
                for (int o = tid; o < F; o += NT)
                    hid[o] = St<T>::rnd(fmaxf(Wl.b_1[o] + gemv_out(part, F, G, o), 0.f));
                team_sync<NT>();
            }
            proj_resid_ln((const T*)Wl.w_2, Wl.b_2, hid, F, Wl.ln2_g, Wl.ln2_b);
        }
    };
    // Encoding of event (t, k) into x / xin (App. D.4 temporal encoding
    // z_i = sin / cos (a_i + b_i t), angle reduced mod 2 pi in fp64, plus the
    // mark embedding); zin = rounded z.  Not synced.
    auto embed = [&](double t, int k) {
        for (int i = tid; i < d; i += NT) {
            const double ang = m.tenc[i] + m.tenc[d + i] * t;
            const double red = fma(-6.283185307179586476925, rint(ang * 0.15915494309189533577), ang);
            float sv, cv;
            sincosf((float)red, &sv, &cv);
            const float z = (i & 1) ? cv : sv;
            const float v = z + m.type_emb[(size_t)k * d + i];
            zin[i] = St<T>::rnd(z);
            x[i] = v;
            xin[i] = St<T>::rnd(v);
        }
    };
    for (int p = nd; p < n; ++p) {  // catch-up over events already emitted
        const size_t so = (size_t)s * ss.n_max + p;
        embed(ss.t[so], min(max(ss.k[so], 0), K - 1));
        team_sync<NT>();
        layers(p);
    }
    if (tid == 0) {
        const long long last = n + a.gamma - 2;  // last position the round encodes
        atomicAdd(&a.st->draft_keys, (unsigned long long)((last + 1) * (last + 2) / 2 - (long long)nd * (nd + 1) / 2));
    }
    const HeadW& H = m.head;
    const int OPh = W <= 32 ? 32 : (W <= 64 ? 64 : 128);
    for (int l = 1; l <= a.gamma; ++l) {
        const int p = n + l - 1;  // index of the drafted event
        // head (Sec. 4.2): e = E h | a = tanh(V_k1 h + b_k1)
        {
            const int G = team_gemv<float, NT>(H.E, 3 * d, H.v_k1, d, x, d, part);
            for (int o = tid; o < 4 * d; o += NT) {
                const float v = gemv_out(part, 4 * d, G, o);
                e[o] = o < 3 * d ? v : tanhf(v + H.b_k1[o - 3 * d]);
            }
            team_sync<NT>();
        }
        // [w logits | mu | log sigma | mark logits] in blocks of OPh outputs;
        // output j reads its own matrix and input segment
        for (int ob = 0; ob < W; ob += OPh) {
            {
                const int G = NT / OPh, o = ob + tid % OPh, g = tid / OPh;
                const int per = (d + G - 1) / G, i0 = g * per, i1 = min(d, i0 + per);
                float acc = 0.f;
                if (o < W) {
                    const float* WT;
                    const float* in;
                    int ld, oo;
                    if (o < M) { WT = H.v_w; in = e; ld = M; oo = o; }
                    else if (o < 2 * M) { WT = H.v_mu; in = e + d; ld = M; oo = o - M; }
                    else if (o < 3 * M) { WT = H.v_s; in = e + 2 * d; ld = M; oo = o - 2 * M; }
                    else { WT = H.v_k2; in = e + 3 * d; ld = K; oo = o - 3 * M; }
                    acc = dot_range<float>(WT, ld, oo, in, i0, i1);
                }
                part[tid] = acc;
            }
            team_sync<NT>();
            if (tid < OPh && ob + tid < W) {
                const int o = ob + tid;
                float v = o < M ? H.b_w[o] : o < 2 * M ? H.b_mu[o - M] : o < 3 * M ? H.b_s[o - 2 * M] : H.b_k2[o - 3 * M];
                for (int gg = 0; gg < NT / OPh; ++gg) v += part[gg * OPh + tid];
                hd[o] = v;
            }
            team_sync<NT>();
        }
        // direct sample: warp 0 the time (component, Box-Muller), warp 1 the
        // mark; both normalise their logits in place
        const size_t so = (size_t)s * ss.n_max + p;
        if (warp < 2) {
            const U4 u = slot_uniforms(P.seed, (uint32_t)s, (uint32_t)p, 0u);
            if (warp == 0) {
                const int z = warp_logsoftmax_pick<2>(hd, M, u.x);
                if (lane == 0) {
                    const float eps = sqrtf(-2.0f * logf(u.y)) * cospif(2.0f * u.z);
                    const float tau = expf(hd[M + z] + expf(hd[2 * M + z]) * eps);
                    const double t = ss.t[so - 1] + (double)tau;
                    ss.tau[so] = tau;
                    ss.t[so] = t;
                    t_new = t;
                }
            } else {
                const int k = warp_logsoftmax_pick<8>(hd + 3 * M, K, u.w);
                if (lane == 0) {
                    ss.k[so] = k;
                    k_new = k;
                }
            }
        }
        team_sync<NT>();
        float* rec = a.heads + ((size_t)s * a.gamma_max + (l - 1)) * W;
        for (int i = tid; i < W; i += NT) rec[i] = hd[i];
        if (l < a.gamma) {
            embed(t_new, k_new);
            team_sync<NT>();
            layers(p);
        }
    }
    pdl_trigger();
}

template <typename T, int DH, bool KVS, bool WS, int NT>
static cudaError_t launch_t(DraftTeamArgs& a, int B, int area, size_t sm, cudaStream_t st) {
    constexpr int TEAMS = WS ? 2 : 1;
    cudaError_t e = cudaFuncSetAttribute(k_draft_team<T, DH, KVS, WS, NT>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    return launch_k(k_draft_team<T, DH, KVS, WS, NT>, dim3((B + TEAMS - 1) / TEAMS), dim3(NT * TEAMS), sm, st, a,
                    area);
}

template <typename T, int DH>
static cudaError_t launch_team(DraftTeamArgs& a, int B, int kvs, int ws, int nt, size_t area, size_t wb,
                               cudaStream_t st) {
    if (ws) return launch_t<T, DH, true, true, 128>(a, B, (int)area, wb + 2 * area, st);
    if (nt == 256) {
        if (kvs) return launch_t<T, DH, true, false, 256>(a, B, (int)area, area, st);
        return launch_t<T, DH, false, false, 256>(a, B, (int)area, area, st);
    }
    if (kvs) return launch_t<T, DH, true, false, 128>(a, B, (int)area, area, st);
    return launch_t<T, DH, false, false, 128>(a, B, (int)area, area, st);
}

int draft_team_supported(const DevModel& m) {
    const int nh = m.nh;
    if (!(nh == 1 || nh == 2 || nh == 4) || !(m.dh == 16 || m.dh == 32)) return 0;
    return m.M <= 64 && m.K <= 256;
}

// The sequence's draft KV is kept in shared memory for the round when that
// still leaves room for two sequences per SM; then, if the model also fits,
// two sequences share a CTA and a staged copy of the model.  Otherwise KV
// and weights are read from HBM/L2.
cudaError_t launch_draft_team(const DevModel& m, const KVCache& kv, const SeqState& ss,
                              const CallParams* dp, int B, int gamma, float* draft_heads,
                              int gamma_max, DevStats* stats, int* err, cudaStream_t st) {
    DraftTeamArgs a{};
    a.m = m; a.kv = kv; a.ss = ss; a.P = dp; a.st = stats; a.heads = draft_heads;
    a.gamma = gamma; a.gamma_max = gamma_max; a.err = err;
    const size_t eb = m.dtype == 1 ? 2 : 4;
    const int W = 3 * m.M + m.K;
    int dev = 0, n_sm = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
    // 256-thread teams when every sequence can have an SM of its own
    // (TPPSD_DRAFT_NT=128|256 forces a size)
    int nt = B <= n_sm ? 256 : 128;
    if (const char* f = getenv("TPPSD_DRAFT_NT")) nt = atoi(f) == 256 ? 256 : 128;
    const size_t fl = sizeof(float) * (12 * (size_t)m.d + m.F + ((W + 3) & ~3) + team_gp_floats(m.d, m.F, nt) +
                                       (size_t)(nt / 32) * 66) + 64;
    const size_t kvb = ((size_t)m.L * 2 * kv.n_max * m.d * eb + 15) & ~(size_t)15;
    // TPPSD_DRAFT_STREAM=<keys>: stream the KV even where it would fit, two
    // stages of that many keys (exercises the ring's wrap-around and ragged
    // last chunk on small cases)
    const char* force = getenv("TPPSD_DRAFT_STREAM");
    const int kvs = !force && kvb + fl <= 110 * 1024;
    size_t ringb = 0;
    if (force) {
        a.ring_nst = 2;
        a.ring_ch = std::max(1, std::min(256, atoi(force)));
        ringb = 2 * (size_t)a.ring_ch * 2 * m.d * eb;
    } else if (!kvs) {
        // streamed KV: as many stages of up to 64 keys as the CTAs that share
        // an SM leave room for (at most 4 resident: the kernel holds 128
        // registers a thread), 2 to 6 stages
        const int per_sm = nt == 256 ? 1 : std::min(4, std::max(1, (B + n_sm - 1) / n_sm));
        const long long budget = std::max(0ll, (long long)(227 * 1024 / per_sm) - 2048 - (long long)fl);
        int ch = 64;
        auto stage = [&](int c) { return (size_t)c * 2 * m.d * eb; };
        while (ch > 16 && 2 * stage(ch) > (size_t)budget) ch /= 2;
        const int nst = (int)std::max<size_t>(2, std::min<size_t>(6, (size_t)budget / stage(ch)));
        a.ring_nst = nst;
        a.ring_ch = ch;
        ringb = nst * stage(ch);
    }
    const size_t area = ((kvs ? kvb : ringb) + fl + 15) & ~(size_t)15;
    const size_t wb = m.t.bytes;  // a whole number of 16-byte chunks
    // two 128-thread teams sharing a staged model, unless each sequence gets
    // its own SM
    const int ws = nt == 128 && kvs && wb % 16 == 0 && wb + 2 * area <= 224 * 1024;
    if (m.dtype == 0) {
        if (m.dh == 16) return launch_team<float, 16>(a, B, kvs, ws, nt, area, wb, st);
        return launch_team<float, 32>(a, B, kvs, ws, nt, area, wb, st);
    }
    if (m.dh == 16) return launch_team<bf16, 16>(a, B, kvs, ws, nt, area, wb, st);
    return launch_team<bf16, 32>(a, B, kvs, ws, nt, area, wb, st);
}


// ---------------------------------------------------------------- lane form
// Draft models with d <= 32 and one or two heads.  Lane i of every warp of
// a sequence's team holds component i of the hidden state, so residual adds,
// LayerNorms and activations run in registers, and each warp computes the
// matrix-vector products it needs itself from the lane-packed model copy
// (chunk c of output j at (c * out + j) * CH: the lanes of a warp read 512
// consecutive bytes per load, CH weights each).  Per layer warp w attends
// with head w % nh over key range w / nh of its key positions (scores kept
// in shared memory, one max and one exponential per key, no rescaling),
// reduces its numerator by a scatter-reduce across lanes and publishes it;
// after one team barrier every warp merges the ranges of every head itself.
// The FFN hidden units are split in quarters (warp w computes quarter w and
// its FFN2 partial; a second barrier sums them).  The draw: warp 0 computes
// the time head and tau, warp 3 the mark head and the mark, then a third
// barrier hands the event to every warp.
//
// Catch-up encodes and drafted events run through one loop body, so the
// code of a drafted event is already in the instruction cache when the
// first draft is drawn.  The uniforms of all gamma draws (and the
// Box-Muller normals) are computed up front, lanes in parallel.  Absolute
// time is carried as a pair of fp32 values (hi + lo, ~48 bits) for the
// temporal encoding, whose angle a_j + b_j t is formed and reduced mod 2 pi
// in that pair arithmetic (FMA-exact products, 2 pi as an fp32 pair); the
// fp64 times written for the target are summed by warp 1 off the critical
// path (fp64 arithmetic is slow on this GPU).  bf16 models also take the
// time head as one folded map [V_w E_1; V_mu E_2; V_s E_3] h (products
// formed in fp64 on the host), a reciprocal square root in the LayerNorms
// and a fast divide in the attention merge; fp32 models keep the unfolded
// head and IEEE operations.

__device__ __forceinline__ float bf_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf_hi(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }

// sum over chunks c < nch of the CH products of output j's chunk c with
// in[c * CH ..] (in: shared, 16-byte aligned; P: lane-packed with OUT outputs)
template <typename TW>
__device__ __forceinline__ float pdot(const TW* __restrict__ P, int OUT, int j, const float* __restrict__ in,
                                      int nch) {
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
    const uint4* w = reinterpret_cast<const uint4*>(P) + j;
    const float4* x = reinterpret_cast<const float4*>(in);
#pragma unroll 4
    for (int c = 0; c < nch; ++c) {
        const uint4 u = w[(size_t)c * OUT];
        if constexpr (sizeof(TW) == 2) {
            const float4 x0 = x[2 * c], x1 = x[2 * c + 1];
            a0 = fmaf(bf_lo(u.x), x0.x, a0);
            a1 = fmaf(bf_hi(u.x), x0.y, a1);
            a2 = fmaf(bf_lo(u.y), x0.z, a2);
            a3 = fmaf(bf_hi(u.y), x0.w, a3);
            a0 = fmaf(bf_lo(u.z), x1.x, a0);
            a1 = fmaf(bf_hi(u.z), x1.y, a1);
            a2 = fmaf(bf_lo(u.w), x1.z, a2);
            a3 = fmaf(bf_hi(u.w), x1.w, a3);
        } else {
            const float4 x0 = x[c];
            a0 = fmaf(__uint_as_float(u.x), x0.x, a0);
            a1 = fmaf(__uint_as_float(u.y), x0.y, a1);
            a2 = fmaf(__uint_as_float(u.z), x0.z, a2);
            a3 = fmaf(__uint_as_float(u.w), x0.w, a3);
        }
    }
    return (a0 + a1) + (a2 + a3);
}

// One halving step of a scatter-reduce over lane pairs (lane, lane ^ OFF):
// the lane with bit OFF set keeps the upper CNT / 2 entries (moved down),
// the other the lower ones, each adding its partner's copy.
template <int CNT, int OFF, int N>
__device__ __forceinline__ void rs_step(float (&v)[N], int lane) {
    const bool up = (lane & OFF) != 0;
#pragma unroll
    for (int i = 0; i < CNT / 2; ++i) {
        const float send = up ? v[i] : v[CNT / 2 + i];
        const float keep = up ? v[CNT / 2 + i] : v[i];
        v[i] = keep + __shfl_xor_sync(FULL, send, OFF);
    }
}
// Sum of v[c] over the 32 lanes; lane receives the total of entry
// (N == 16 ? lane >> 1 : lane).
template <int N>
__device__ __forceinline__ float warp_scatter_sum(float (&v)[N], int lane) {
    static_assert(N == 16 || N == 32, "16 or 32 entries");
    if constexpr (N == 32) rs_step<32, 16>(v, lane);
    rs_step<16, N == 32 ? 8 : 16>(v, lane);
    rs_step<8, N == 32 ? 4 : 8>(v, lane);
    rs_step<4, N == 32 ? 2 : 4>(v, lane);
    rs_step<2, N == 32 ? 1 : 2>(v, lane);
    if constexpr (N == 16) v[0] += __shfl_xor_sync(FULL, v[0], 1);
    return v[0];
}

// LayerNorm of the d values held by lanes < d (v; others ignored); FAST
// takes the reciprocal square root instruction instead of 1 / sqrt.
template <bool FAST>
__device__ __forceinline__ float lane_ln(float v, int lane, float inv_d, int d, const float* g, const float* b) {
    const bool live = lane < d;
    const float mean = warp_sum(live ? v : 0.f) * inv_d;
    const float c = live ? v - mean : 0.f;
    const float var = warp_sum(c * c) * inv_d + LN_EPS;
    const float inv = FAST ? rsqrtf(var) : 1.0f / sqrtf(var);
    return live ? c * inv * g[lane] + b[lane] : 0.f;
}

// Log-softmax of v[0..n) (shared, n <= NMAX) in place, and the smallest
// index whose running sum of probabilities reaches u * total, with every
// sum taken in index order (the same rule as warp_logsoftmax_pick, whose
// scans sum in tree order).  By a whole warp: lane i < n evaluates the
// exponentials of value i, and every lane forms the ordered sums itself
// from shuffled copies, so all lanes hold the same sums and the same pick.
// Ends with __syncwarp.
template <int NMAX>
__device__ __forceinline__ int lane_logsoftmax_pick(float* v, int n, float u) {
    const int lane = threadIdx.x & 31;
    const float xi = lane < n ? v[lane] : -INFINITY;
    float mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < NMAX; ++i) mx = fmaxf(mx, __shfl_sync(FULL, xi, i));
    const float ei = lane < n ? expf(xi - mx) : 0.f;
    float sm = 0.f;
#pragma unroll
    for (int i = 0; i < NMAX; ++i) sm += __shfl_sync(FULL, ei, i);
    const float lz = mx + logf(sm);
    float pi = 0.f;
    if (lane < n) {
        const float xn = xi - lz;
        v[lane] = xn;
        pi = expf(xn);
    }
    float pr[NMAX], tot = 0.f;
#pragma unroll
    for (int i = 0; i < NMAX; ++i) {
        pr[i] = __shfl_sync(FULL, pi, i);
        tot += pr[i];
    }
    const float target = u * tot;
    float run = 0.f;
    int pick = n - 1;
    bool found = false;
#pragma unroll
    for (int i = 0; i < NMAX; ++i) {
        run += pr[i];
        if (!found && i < n && run >= target) {
            pick = i;
            found = true;
        }
    }
    __syncwarp();
    return pick;
}

// fp32 pair arithmetic (hi + lo): exact sum of two floats, and sum of a
// pair and a float (Knuth's two-sum; Dekker's fast two-sum for |a| >= |b|).
struct F2 { float h, l; };
__device__ __forceinline__ F2 two_sum(float a, float b) {
    const float s = a + b, bb = s - a;
    return {s, (a - (s - bb)) + (b - bb)};
}
__device__ __forceinline__ F2 fast_two_sum(float a, float b) {
    const float s = a + b;
    return {s, b - (s - a)};
}
__device__ __forceinline__ F2 f2_add(F2 a, float b) {
    const F2 s = two_sum(a.h, b);
    return fast_two_sum(s.h, s.l + a.l);
}
__device__ __forceinline__ F2 f2_from_double(double t) {
    const float h = __double2float_rn(t);
    return {h, __double2float_rn(t - (double)h)};
}
// (a + b t) mod 2 pi in [-pi, pi] as fp32, from fp32 pairs a, b, t: the
// product and sums in pair arithmetic, then k = rint(angle / 2 pi) removed
// with 2 pi = P_HI + P_LO (k * P_HI split exactly by an FMA; the angle minus
// k * P_HI is exact because both lie within a factor of two).
__device__ __forceinline__ float reduced_angle(F2 a, F2 b, F2 t) {
    const float P_HI = 6.28318548202514648f, P_LO = -1.74845553e-7f, INV = 0.159154943091895336f;
    const float p = b.h * t.h;
    float e = fmaf(b.h, t.h, -p);
    e = fmaf(b.h, t.l, e);
    e = fmaf(b.l, t.h, e);
    const F2 s = two_sum(a.h, p);
    const F2 ang = fast_two_sum(s.h, s.l + (e + a.l));
    const float k = rintf(ang.h * INV);
    const float q = k * P_HI, qe = fmaf(k, P_HI, -q);
    float r = ang.h - q;
    r = r - qe;
    r = r + ang.l;
    return fmaf(-k, P_LO, r);
}

// Shared-memory floats of one team besides its KV: head row, attention
// partials (two sets of 4 warps x (max, sum, -, -, 32 numerators)), FFN2
// partials (4 x 32), the drawn event (t hi, t lo, tau, k), then per warp:
// input vector (64), attention output / fp32 hidden state (32), FFN quarter
// (64), head activations (96), query (32), draw constants (2 G) and the key
// scores (sc).
__host__ __device__ inline int lane_warp_floats(int G, int sc) { return 288 + 2 * G + sc; }
__host__ __device__ inline int lane_team_floats(int W, int G, int sc) {
    return ((W + 3) & ~3) + 2 * 4 * 36 + 128 + 4 + 4 * lane_warp_floats(G, sc);
}

// Pairs i0, i0 + stride, ... of the target's embedding of verify row r
// (event (t, k) at position pos of sequence s, THP or SAHP layout): the
// same arithmetic as the forward's embedding kernel, whose launch the lane
// form replaces.  live == false writes the inactive row (zeros, s = -1).
template <typename T>
__device__ __forceinline__ void draft_embed_row(const DraftEmbed& e, int r, int s, int pos, double t, int k,
                                                bool live, int i0, int stride) {
    const int half = e.d / 2;
    k = min(max(k, 0), e.K - 1);
    T* xb = (T*)e.xb;
    for (int i = i0; i < half; i += stride) {
        float z0 = 0.f, z1 = 0.f, e0 = 0.f, e1 = 0.f;
        if (live) {
            tenc_pair_of(e.tenc, e.d, e.paired, t, i, &z0, &z1);
            e0 = e.type_emb[(size_t)k * e.d + 2 * i];
            e1 = e.type_emb[(size_t)k * e.d + 2 * i + 1];
        }
        const size_t xo = (size_t)r * e.d + 2 * i;
        e.x[xo] = z0 + e0;
        e.x[xo + 1] = z1 + e1;
        St<T>::st(xb + xo, z0 + e0);
        St<T>::st(xb + xo + 1, z1 + e1);
    }
    if (i0 == 0) {
        e.row_seq[r] = live ? s : -1;
        e.row_pos[r] = pos;
    }
}

// D: the draft width (16 or 32), a compile-time constant so that the
// product loops, lane predicates and head splits are fixed.
template <typename T, int DH, int D>
__global__ void __launch_bounds__(256) k_draft_lane(DraftTeamArgs a, int area_bytes, int sc_stride, int g_stride) {
    extern __shared__ __align__(16) char smem[];
    __shared__ uint64_t wbar;
    constexpr bool BF = sizeof(T) == 2;
    constexpr int CH = 16 / sizeof(T);
    const DevModelT& mp = a.m.p;
    const char* gb = mp.base;
    const uint32_t wb = (uint32_t)mp.bytes;
    // the model is never written by a sampling kernel: stage it while the
    // previous kernel of the stream finishes
    if (threadIdx.x == 0) {
        mbar_init(&wbar, 1);
        mbar_fence_init();
        mbar_arrive_expect_tx(&wbar, wb);
        bulk_load(smem, gb, wb, &wbar);
    }
    pdl_wait();
    const int team = threadIdx.x >> 7;
    const int s = blockIdx.x * 2 + team;
    const int tid = threadIdx.x & 127, warp = tid >> 5, lane = tid & 31;
    constexpr int d = D, NH = D / DH;
    const int F = a.m.F, M = a.m.M, K = a.m.K, W = 3 * M + K, L = a.m.L;
    const int n_max = a.kv.n_max;
    const CallParams& P = *a.P;
    const SeqState& ss = a.ss;
    const bool live = s < P.B && !ss.done[s];
    char* area = smem + wb + (size_t)team * area_bytes;
    const size_t kvb = ((size_t)L * 2 * n_max * d * sizeof(T) + 15) & ~(size_t)15;
    T* kvs = (T*)area;
    uint64_t* bar = (uint64_t*)(area + kvb);
    int n = 0, nd = 0;
    if (live) {
        n = ss.n_emit[s];
        nd = ss.n_draft[s];
    }
    auto gk = [&](int l, int w) -> T* {
        return (T*)(w ? a.kv.v : a.kv.k) + (((size_t)l * a.kv.Bmax + s) * NH) * (size_t)n_max * DH;
    };
    auto sk = [&](int l, int w) -> T* { return kvs + (((size_t)l * 2 + w) * NH) * (size_t)n_max * DH; };
    if (tid == 0 && live && nd > 0) {
        // the sequence's draft KV: each (layer, K/V, head) block of positions
        // 0..nd-1 is contiguous in HBM
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
    const bool emb = a.emb.x != nullptr;
    const int q = a.gamma + 1;  // verify rows per sequence
    if (!live) {
        if (emb && s < P.B) {  // the sequence's verify rows, inactive
            const int ne = ss.n_emit[s];
            for (int l = 0; l < q; ++l)
                draft_embed_row<T>(a.emb, s * q + l, s, ne - 1 + l, 0.0, 0, false, tid, 128);
        }
        // a CTA may not exit while the model copy still writes its shared memory
        mbar_wait(&wbar, 0, a.err, 14);
        return;  // the rest synchronises within the team only
    }
    constexpr int S = 4 / NH;
    const int hw = warp % NH, spw = warp / NH;  // this warp's head and key range
    const bool att_enc = a.m.enc == 2;
    const float inv_d = 1.0f / (float)d;
    float* hd = (float*)(area + kvb + 16);
    float* red = hd + ((W + 3) & ~3);  // [2][4][36]
    float* part = red + 2 * 4 * 36;    // [4][32]
    float* ev = part + 128;            // t hi, t lo, tau, k (int bits)
    float* mine = ev + 4 + warp * lane_warp_floats(g_stride, sc_stride);
    float* v_in = mine;        // [zin | xin] (AttNHP) or xin
    float* v_att = mine + 64;  // attention output; fp32 hidden state for the head
    float* v_hid = mine + 96;  // this warp's FFN quarter
    float* v_e = mine + 160;   // head activations
    float* v_q = mine + 256;   // query of this warp's head
    float* v_rng = mine + 288; // draw constants of the gamma events
    float* sc = v_rng + 2 * g_stride;  // scores of this warp's keys
    auto sm = [&](const void* g) -> const char* { return smem + ((const char*)g - gb); };
    const int gamma = a.gamma, p_last = n + gamma - 1;
    // draw constants: warp 0 (u_comp, eps) and warp 3 (u_mark) of draft l at
    // position n + l, from the block-0 slot of that position
    if (warp == 0 || warp == 3)
        for (int l = lane; l < gamma; l += 32) {
            const U4 u = slot_uniforms(P.seed, (uint32_t)s, (uint32_t)(n + l), 0u);
            if (warp == 0) {
                v_rng[2 * l] = u.x;
                v_rng[2 * l + 1] = sqrtf(-2.0f * logf(u.y)) * cospif(2.0f * u.z);
            } else {
                v_rng[2 * l] = u.w;
            }
        }
    // catch-up events (t, k) read before the waits
    double t_cu[2] = {0.0, 0.0};
    int k_cu[2] = {0, 0};
    for (int i = 0; i < 2 && nd + i < n; ++i) {
        const size_t so = (size_t)s * ss.n_max + nd + i;
        t_cu[i] = ss.t[so];
        k_cu[i] = min(max(ss.k[so], 0), K - 1);
    }
    double t64 = ss.t[(size_t)s * ss.n_max + n - 1];  // fp64 time of the last event (warp 1)
    int k_emb = 0;  // mark of the last drawn event (warp 1)
    if (tid == 0) {  // its pair form, which the first draft adds to
        const F2 t2 = f2_from_double(t64);
        ev[0] = t2.h;
        ev[1] = t2.l;
    }
    if (emb)  // verify row 0: the last emitted event, at position n - 1
        draft_embed_row<T>(a.emb, s * q, s, n - 1, t64, min(max(ss.k[(size_t)s * ss.n_max + n - 1], 0), a.emb.K - 1),
                           true, tid, 128);
    mbar_wait(&wbar, 0, a.err, 14);
    if (nd > 0) mbar_wait(bar, 0, a.err, 12);
    const float* type_emb = (const float*)sm(mp.type_emb);
    const float* tff = (const float*)sm(mp.tenc_ff);
    F2 ta{0.f, 0.f}, tb{0.f, 0.f};  // a_lane, b_lane of the encoding
    if (lane < d) {
        ta = {tff[lane], tff[d + lane]};
        tb = {tff[2 * d + lane], tff[3 * d + lane]};
    }
    const float scale = 1.4426950408889634f / sqrtf((float)DH);
    float x = 0.f;
    __syncwarp();
    for (int p = nd;; ++p) {
        F2 tp;
        int kp;
        if (p >= n) {
            // draw event p from the head of the hidden state x of p - 1
            // (Sec. 4.2): z ~ Cat(w), tau = exp(mu_z + sigma_z eps); k ~ f
            const int l = p - n;
            const size_t so = (size_t)s * ss.n_max + p;
            const HeadW& H = mp.head;
            if (warp == 0) {
                if (lane < d) v_att[lane] = x;
                __syncwarp();
                if constexpr (BF) {
                    const float* ht = (const float*)sm(mp.head_t);
                    const float* htb = (const float*)sm(mp.head_tb);
                    for (int o = lane; o < 3 * M; o += 32) hd[o] = pdot<float>(ht, 3 * M, o, v_att, d / 4) + htb[o];
                } else {
                    const float* E = (const float*)sm(H.E);
                    if (lane < d) {
#pragma unroll
                        for (int r = 0; r < 3; ++r)
                            v_e[r * d + lane] = pdot<float>(E, 3 * d, r * d + lane, v_att, d / 4);
                    }
                    __syncwarp();
                    for (int o = lane; o < 3 * M; o += 32) {
                        const int seg = o / M, jj = o - seg * M;
                        const float* V = (const float*)sm(seg == 0 ? H.v_w : seg == 1 ? H.v_mu : H.v_s);
                        const float* bb = (const float*)sm(seg == 0 ? H.b_w : seg == 1 ? H.b_mu : H.b_s);
                        hd[o] = pdot<float>(V, M, jj, v_e + seg * d, d / 4) + bb[jj];
                    }
                }
                __syncwarp();
                int z;
                if (M <= 8) {
                    z = lane_logsoftmax_pick<8>(hd, M, v_rng[2 * l]);
                } else {
                    z = warp_logsoftmax_pick<2>(hd, M, v_rng[2 * l]);
                }
                if (lane == 0) {
                    const float tau = expf(hd[M + z] + expf(hd[2 * M + z]) * v_rng[2 * l + 1]);
                    const F2 tn = f2_add(F2{ev[0], ev[1]}, tau);
                    ev[0] = tn.h;
                    ev[1] = tn.l;
                    ev[2] = tau;
                    ss.tau[so] = tau;
                }
            } else if (warp == 3) {
                if (lane < d) v_att[lane] = x;
                __syncwarp();
                if (lane < d)
                    v_e[lane] = tanhf(pdot<float>((const float*)sm(H.v_k1), d, lane, v_att, d / 4) +
                                      ((const float*)sm(H.b_k1))[lane]);
                __syncwarp();
                const float* V2 = (const float*)sm(H.v_k2);
                const float* b2 = (const float*)sm(H.b_k2);
                for (int o = lane; o < K; o += 32) hd[3 * M + o] = pdot<float>(V2, K, o, v_e, d / 4) + b2[o];
                __syncwarp();
                int k;
                if (K <= 8) {
                    k = lane_logsoftmax_pick<8>(hd + 3 * M, K, v_rng[2 * l]);
                } else {
                    k = warp_logsoftmax_pick<8>(hd + 3 * M, K, v_rng[2 * l]);
                }
                if (lane == 0) {
                    ss.k[so] = k;
                    ev[3] = __int_as_float(k);
                }
            } else if (warp == 1 && emb && l >= 1) {
                // idle while warps 0 and 3 draw: the target's verify row of the
                // previous draft (row l, position p - 1)
                draft_embed_row<T>(a.emb, s * q + l, s, p - 1, t64, k_emb, true, lane, 32);
            }
            team_sync();
            tp = {ev[0], ev[1]};
            kp = __float_as_int(ev[3]);
            if (warp == 1) {
                float* rec = a.heads + ((size_t)s * a.gamma_max + l) * W;
                for (int i = lane; i < W; i += 32) rec[i] = hd[i];
                t64 += (double)ev[2];  // the fp64 time of the event, as the target reads it
                k_emb = kp;
                if (lane == 0) ss.t[so] = t64;
            }
            if (p == p_last) {
                if (warp == 1 && emb)  // the last draft's verify row (row gamma)
                    draft_embed_row<T>(a.emb, s * q + q - 1, s, p, t64, k_emb, true, lane, 32);
                break;
            }
        } else {
            const int i = p - nd;
            double t;
            if (i < 2) {
                t = i == 0 ? t_cu[0] : t_cu[1];
                kp = i == 0 ? k_cu[0] : k_cu[1];
            } else {
                const size_t so = (size_t)s * ss.n_max + p;
                t = ss.t[so];
                kp = min(max(ss.k[so], 0), K - 1);
            }
            tp = f2_from_double(t);
        }
        // ---- encode event p: temporal encoding z_i = sin / cos (a_i + b_i t)
        // (App. D.4) plus the mark embedding
        if (lane < d) {
            float sv, cv;
            sincosf(reduced_angle(ta, tb, tp), &sv, &cv);
            const float z = (lane & 1) ? cv : sv;
            x = z + type_emb[(size_t)kp * d + lane];
            if (att_enc) {
                v_in[lane] = St<T>::rnd(z);
                v_in[d + lane] = St<T>::rnd(x);
            } else {
                v_in[lane] = St<T>::rnd(x);
            }
        }
        __syncwarp();
        // key ranges of length per, the last one ~32 keys shorter: the warp
        // whose range holds key p also computes k and v of p
        const int nk = p + 1, per = (nk + 32 + S - 1) / S, lo = spw * per, hi = min(nk, lo + per);
        const bool writer = spw == p / per;
        for (int l = 0; l < L; ++l) {
            const LayerW& Wl = mp.layer[l];
            const T* wqkv = (const T*)sm(Wl.w_qkv);
            const float* bqkv = (const float*)sm(Wl.b_qkv);
            const int nin = (att_enc ? 2 * d : d) / CH;
            // q of head hw; the writer also appends k and v at position p
            for (int o = lane; o < (writer ? 3 * DH : DH); o += 32) {
                const int part3 = o / DH, c = o - part3 * DH, row = part3 * d + hw * DH + c;
                const float v = St<T>::rnd(pdot<T>(wqkv, 3 * d, row, v_in, nin) + bqkv[row]);
                if (part3 == 0) {
                    v_q[c] = v * scale;
                } else {
                    const size_t off = ((size_t)hw * n_max + p) * DH + c;
                    St<T>::st(gk(l, part3 - 1) + off, v);
                    St<T>::st(sk(l, part3 - 1) + off, v);
                }
            }
            __syncwarp();
            // attention of head hw over keys lo..hi-1 (exp2 units)
            float q[DH];
#pragma unroll
            for (int c = 0; c < DH; ++c) q[c] = v_q[c];
            const T* kb = sk(l, 0) + (size_t)hw * n_max * DH;
            const T* vb = sk(l, 1) + (size_t)hw * n_max * DH;
            // keys j and j + 32 of a lane per iteration: both rows are loaded
            // before either is used (the second is a repeat of the first
            // when j + 32 is past the range, and its terms are dropped)
            float mx = -INFINITY;
#pragma unroll 1
            for (int j = lo + lane; j < hi; j += 64) {
                const bool two = j + 32 < hi;
                float kr[DH], kr2[DH];
                load_row16<T, DH>(kb + (size_t)j * DH, kr);
                load_row16<T, DH>(kb + (size_t)(two ? j + 32 : j) * DH, kr2);
                float s0 = 0.f, s1 = 0.f, t0 = 0.f, t1 = 0.f;
#pragma unroll
                for (int c = 0; c < DH; c += 2) {
                    s0 = fmaf(q[c], kr[c], s0);
                    s1 = fmaf(q[c + 1], kr[c + 1], s1);
                    t0 = fmaf(q[c], kr2[c], t0);
                    t1 = fmaf(q[c + 1], kr2[c + 1], t1);
                }
                const float sv = s0 + s1, sv2 = t0 + t1;
                sc[j - lo] = sv;
                mx = fmaxf(mx, sv);
                if (two) {
                    sc[j + 32 - lo] = sv2;
                    mx = fmaxf(mx, sv2);
                }
            }
            mx = warp_max(mx);
            float ll = 0.f, o[DH];
#pragma unroll
            for (int c = 0; c < DH; ++c) o[c] = 0.f;
#pragma unroll 1
            for (int j = lo + lane; j < hi; j += 64) {
                const bool two = j + 32 < hi;
                const float pj = exp2f(sc[j - lo] - mx);
                const float pj2 = two ? exp2f(sc[j + 32 - lo] - mx) : 0.f;
                float vr[DH], vr2[DH];
                load_row16<T, DH>(vb + (size_t)j * DH, vr);
                load_row16<T, DH>(vb + (size_t)(two ? j + 32 : j) * DH, vr2);
                ll += pj;
                ll += pj2;
#pragma unroll
                for (int c = 0; c < DH; ++c) o[c] = fmaf(pj2, vr2[c], fmaf(pj, vr[c], o[c]));
            }
            ll = warp_sum(ll);
            const float oc = warp_scatter_sum<DH>(o, lane);
            float* rw = red + ((l & 1) * 4 + warp) * 36;
            if (lane == 0) {
                rw[0] = mx;
                rw[1] = ll;
            }
            if (DH == 32 || !(lane & 1)) rw[4 + (DH == 16 ? lane >> 1 : lane)] = oc;
            team_sync();
            // merge the key ranges of head lane / DH for output component lane
            float at = 0.f;
            if (lane < d) {
                const int hj = lane / DH, c = lane - hj * DH;
                const float* rb = red + (l & 1) * 4 * 36;
                float Mx = -INFINITY;
                for (int sp = 0; sp < S; ++sp) Mx = fmaxf(Mx, rb[(sp * NH + hj) * 36]);
                float Lx = 0.f, Ox = 0.f;
                for (int sp = 0; sp < S; ++sp) {
                    const float* src = rb + (sp * NH + hj) * 36;
                    if (src[0] == -INFINITY) continue;
                    const float e = exp2f(src[0] - Mx);
                    Lx += src[1] * e;
                    Ox += src[4 + c] * e;
                }
                if (att_enc) at = Ox / (Lx + exp2f(-Mx));
                else at = St<T>::rnd(BF ? __fdividef(Ox, Lx) : Ox / Lx);
            }
            if (att_enc) {  // AttNHP (App. D.4): h <- h + tanh(a), no projection or FFN
                if (lane < d) {
                    x += tanhf(at);
                    v_in[d + lane] = St<T>::rnd(x);
                }
                __syncwarp();
                continue;
            }
            // x = LN1(x + W_o a + b_o)
            if (lane < d) v_att[lane] = at;
            __syncwarp();
            float y = 0.f;
            if (lane < d) y = pdot<T>((const T*)sm(Wl.w_o), d, lane, v_att, d / CH) + ((const float*)sm(Wl.b_o))[lane];
            x = lane_ln<BF>(x + y, lane, inv_d, d, (const float*)sm(Wl.ln1_g), (const float*)sm(Wl.ln1_b));
            if (lane < d) v_in[lane] = St<T>::rnd(x);
            __syncwarp();
            // FFN quarter of this warp: hidden units f0 .. f0 + F/4 - 1
            const int Fq = F >> 2, f0 = warp * Fq;
            const T* w1 = (const T*)sm(Wl.w_1);
            const float* b1 = (const float*)sm(Wl.b_1);
            for (int jj = lane; jj < Fq; jj += 32)
                v_hid[jj] = St<T>::rnd(fmaxf(pdot<T>(w1, F, f0 + jj, v_in, d / CH) + b1[f0 + jj], 0.f));
            __syncwarp();
            if (lane < d)
                part[warp * 32 + lane] =
                    pdot<T>((const T*)sm(Wl.w_2) + (size_t)(f0 / CH) * d * CH, d, lane, v_hid, Fq / CH);
            team_sync();
            // x = LN2(x + W_2 relu(.) + b_2)
            float y2 = 0.f;
            if (lane < d)
                y2 = ((const float*)sm(Wl.b_2))[lane] +
                     ((part[lane] + part[32 + lane]) + (part[64 + lane] + part[96 + lane]));
            x = lane_ln<BF>(x + y2, lane, inv_d, d, (const float*)sm(Wl.ln2_g), (const float*)sm(Wl.ln2_b));
            if (lane < d) v_in[lane] = St<T>::rnd(x);
            __syncwarp();
        }
    }
    if (tid == 0) {
        const long long last = n + gamma - 2;  // last position the round encodes
        atomicAdd(&a.st->draft_keys, (unsigned long long)((last + 1) * (last + 2) / 2 - (long long)nd * (nd + 1) / 2));
    }
    pdl_trigger();
}

// Shared-memory bytes of one team of the lane form (0: the shape is not
// covered).
static size_t lane_area(const DevModel& m, int n_max, int gamma_max, int* sc_out, int* g_out) {
    const int CH = m.dtype == 1 ? 8 : 4;
    const bool shape = (m.nh == 1 && (m.dh == 16 || m.dh == 32)) || (m.nh == 2 && m.dh == 16);  // d = 16 or 32
    if (!shape || m.d % CH || m.M > 64 || m.K > 256 || m.L < 1) return 0;
    if (m.enc != 2 && (m.F % (4 * CH) || m.F > 256)) return 0;
    const size_t eb = m.dtype == 1 ? 2 : 4;
    const int S = 4 / m.nh;
    const int sc = (((n_max + 32 + S - 1) / S) + 3) & ~3, G = (gamma_max + 3) & ~3;
    const size_t kvb = ((size_t)m.L * 2 * n_max * m.d * eb + 15) & ~(size_t)15;
    if (sc_out) *sc_out = sc;
    if (g_out) *g_out = G;
    return kvb + 16 + sizeof(float) * (size_t)lane_team_floats(3 * m.M + m.K, G, sc);
}

int draft_lane_supported(const DevModel& m, int n_max, int gamma_max) {
    const size_t area = lane_area(m, n_max, gamma_max, nullptr, nullptr);
    if (!area || m.p.bytes % 16 || !m.p.tenc_ff) return 0;
    return m.p.bytes + 2 * area <= 224 * 1024;
}

cudaError_t launch_draft_lane(const DevModel& m, const KVCache& kv, const SeqState& ss,
                              const CallParams* dp, int B, int gamma, float* draft_heads,
                              int gamma_max, DevStats* stats, int* err, cudaStream_t st,
                              const DraftEmbed* emb) {
    DraftTeamArgs a{};
    a.m = m; a.kv = kv; a.ss = ss; a.P = dp; a.st = stats; a.heads = draft_heads;
    a.gamma = gamma; a.gamma_max = gamma_max; a.err = err;
    if (emb) a.emb = *emb;
    int sc = 0, G = 0;
    const size_t area = lane_area(m, kv.n_max, gamma_max, &sc, &G);
    const size_t sm = m.p.bytes + 2 * area;
    auto go = [&](auto kern) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
        if (e != cudaSuccess) return e;
        return launch_k(kern, dim3((B + 1) / 2), dim3(256), sm, st, a, (int)area, sc, G);
    };
    if (m.d == 16) return m.dtype == 0 ? go(k_draft_lane<float, 16, 16>) : go(k_draft_lane<bf16, 16, 16>);
    if (m.dtype == 0) return m.dh == 16 ? go(k_draft_lane<float, 16, 32>) : go(k_draft_lane<float, 32, 32>);
    return m.dh == 16 ? go(k_draft_lane<bf16, 16, 32>) : go(k_draft_lane<bf16, 32, 32>);
}

}  // namespace tppsd
