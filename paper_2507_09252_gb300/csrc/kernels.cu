// Kernels of the TPP-SD sampler (arxiv 2507.09252) for GB300 (sm_103a).
//
// One sampling round of Alg. 1 is: the draft kernel (gamma draft events per
// sequence, Sec. 4.3 "Drafting": k_draft_team in draft.cu, or k_draft here
// for shapes it does not cover) -> batched target forward over gamma+1
// positions per sequence (Sec. 4.3 "Verification"; tensor-core GEMMs in
// gemm_tc.cu and attention in attn.cu for bf16 models) -> heads (fp32 GEMM
// + k_head_out) -> k_verify_epilogue (ratio tests, first rejection,
// Theorem-1 / Eq. 4 resampling, commit and cache rollback) ->
// k_round_control.
#include <math.h>
#include <stdlib.h>

#include <algorithm>

#include <cuda_fp16.h>

#include "common.cuh"
#include "engine.h"
#include "tc_ptx.cuh"

namespace tppsd {

// ======================================================================
// small helpers
// ======================================================================
__device__ __forceinline__ size_t kv_index(const KVCache& kv, int nh, int dh, int layer, int s,
                                           int h, int pos) {
    return ((((size_t)layer * kv.Bmax + s) * nh + h) * (size_t)kv.n_max + pos) * (size_t)dh;
}

template <typename T>
__device__ __forceinline__ void load_row(const T* p, float* out, int n) {
    for (int c = 0; c < n; ++c) out[c] = St<T>::ld(p + c);
}

// Temporal encoding (App. D.4: z_j = sin / cos (a_j + b_j t) for even / odd
// j) of dimensions 2i, 2i+1.  THP and AttNHP pairs share one angle (one
// sincos); SAHP's dimensions have their own.
__device__ __forceinline__ void tenc_pair(const DevModel& m, double t, int i, float* z0, float* z1) {
    tenc_pair_of(m.tenc, m.d, m.tenc_paired, t, i, z0, z1);
}

// Temporal encoding + type embedding (Sec. 4.2) of pair i.  Marks outside
// 0..K-1 are clamped into range (the row gather stays in bounds).
__device__ __forceinline__ void embed_pair(const DevModel& m, double t, int k, int i, float* z0,
                                           float* z1) {
    k = min(max(k, 0), m.K - 1);
    tenc_pair(m, t, i, z0, z1);
    *z0 += m.type_emb[(size_t)k * m.d + 2 * i];
    *z1 += m.type_emb[(size_t)k * m.d + 2 * i + 1];
}

// ======================================================================
// batched forward: embed, GEMM (+epilogues), attention, LayerNorm, head
// ======================================================================
template <typename T>
__global__ void k_embed(DevModel m, SeqState ss, RowSpec rs, Work w) {
    pdl_wait();
    const int half = m.d / 2;
    const long long total = (long long)rs.count * half;
    T* xb = (T*)w.xb;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const int r = (int)(idx / half), i = (int)(idx % half);
        int s, pos;
        bool active;
        if (rs.mode == ROWS_STEP) {
            s = r / rs.q;
            active = !ss.done[s];
            pos = ss.n_emit[s] - 1 + r % rs.q;
        } else {
            const long long g = rs.g0 + (long long)r;
            s = (int)(g / rs.q);
            pos = (int)(g % rs.q);
            active = true;
        }
        if (i == 0) {
            w.row_seq[r] = active ? s : -1;
            w.row_pos[r] = pos;
        }
        float z0 = 0.f, z1 = 0.f, e0 = 0.f, e1 = 0.f;
        if (active) {
            const size_t o = (size_t)s * ss.n_max + pos;
            const int k = min(max(ss.k[o], 0), m.K - 1);
            tenc_pair(m, ss.t[o], i, &z0, &z1);
            e0 = m.type_emb[(size_t)k * m.d + 2 * i];
            e1 = m.type_emb[(size_t)k * m.d + 2 * i + 1];
        }
        const size_t xo = (size_t)r * m.d + 2 * i;
        w.x[xo] = z0 + e0;
        w.x[xo + 1] = z1 + e1;
        if (m.enc == 2) {  // AttNHP: rows [z | h] (the QKV input of every layer)
            const size_t zo = (size_t)r * 2 * m.d + 2 * i;
            St<T>::st(xb + zo, z0);
            St<T>::st(xb + zo + 1, z1);
            St<T>::st(xb + zo + m.d, z0 + e0);
            St<T>::st(xb + zo + m.d + 1, z1 + e1);
        } else {
            St<T>::st(xb + xo, z0 + e0);
            St<T>::st(xb + xo + 1, z1 + e1);
        }
    }
    pdl_trigger();
}

enum { EPI_QKV = 0, EPI_RELU = 1, EPI_RESID = 2, EPI_F32 = 3 };

template <typename T>
struct GemmArgs {
    const T* A;          // [R][K]
    const T* W;          // [N][K]
    const float* bias;   // [N]
    int R, N, K;
    // EPI_QKV (v_f16: V stored as fp16 of the storage-type value)
    T* q_out; T* kc; T* vc; const int* row_seq; const int* row_pos;
    int d, nh, dh, layer, Bmax, n_max, v_f16;
    // EPI_RELU: T out [R][N]; EPI_RESID: float out [R][N] = acc + b + resid
    T* out_t; float* out_f; const float* resid;
};

// SIMT tiled GEMM, 64x64 tile, 256 threads, 4x4 outputs per thread, fp32
// accumulation, Y = A W^T + b with a fused epilogue.
template <typename T, int EPI>
__global__ void __launch_bounds__(256) k_gemm(GemmArgs<T> a) {
    constexpr int BM = 64, BN = 64, BK = 32;
    __shared__ __align__(16) float As[BK][BM + 4];
    __shared__ __align__(16) float Ws[BK][BN + 4];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int row0 = blockIdx.y * BM, col0 = blockIdx.x * BN;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    const int lr = tid >> 2, kc = (tid & 3) * 8;
    for (int k0 = 0; k0 < a.K; k0 += BK) {
        const int gr = row0 + lr, gc = col0 + lr;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int gk = k0 + kc + e;
            As[kc + e][lr] = (gr < a.R && gk < a.K) ? St<T>::ld(a.A + (size_t)gr * a.K + gk) : 0.f;
            Ws[kc + e][lr] = (gc < a.N && gk < a.K) ? St<T>::ld(a.W + (size_t)gc * a.K + gk) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < BK; ++kk) {
            const float4 av = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
            const float4 wv = *reinterpret_cast<const float4*>(&Ws[kk][tx * 4]);
            const float ar[4] = {av.x, av.y, av.z, av.w}, wr[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(ar[i], wr[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int r = row0 + ty * 4 + i;
        if (r >= a.R) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int c = col0 + tx * 4 + j;
            if (c >= a.N) continue;
            const float v = acc[i][j] + a.bias[c];
            if (EPI == EPI_QKV) {
                const int which = c / a.d, cc = c - which * a.d;
                if (which == 0) {
                    St<T>::st(a.q_out + (size_t)r * a.d + cc, v);
                } else {
                    const int s = a.row_seq[r];
                    if (s < 0) continue;
                    const int h = cc / a.dh, e = cc - h * a.dh;
                    const size_t o = ((((size_t)a.layer * a.Bmax + s) * a.nh + h) * (size_t)a.n_max +
                                      a.row_pos[r]) * a.dh + e;
                    if (which == 2 && a.v_f16)  // exact: a bf16 value in the fp16 range
                        reinterpret_cast<__half*>(a.vc)[o] = __float2half_rn(St<T>::rnd(v));
                    else
                        St<T>::st((which == 1 ? a.kc : a.vc) + o, v);
                }
            } else if (EPI == EPI_RELU) {
                St<T>::st(a.out_t + (size_t)r * a.N + c, fmaxf(v, 0.f));
            } else if (EPI == EPI_F32) {
                a.out_f[(size_t)r * a.N + c] = v;
            } else {
                a.out_f[(size_t)r * a.N + c] = v + a.resid[(size_t)r * a.N + c];
            }
        }
    }
}

// LayerNorm of y (fp32) into x (fp32) and its storage-type copy xb; one warp per row.
template <typename T>
__global__ void k_layernorm(const float* y, const float* g, const float* b, float* x, T* xb, int R,
                            int d) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = blockIdx.x * (blockDim.x >> 5) + warp;
    if (r >= R) return;
    float v[MAX_D / 32];
    float sum = 0.f;
#pragma unroll
    for (int j = 0; j < MAX_D / 32; ++j) {
        const int i = lane + 32 * j;
        v[j] = i < d ? y[(size_t)r * d + i] : 0.f;
        sum += v[j];
    }
    const float mean = warp_sum(sum) / d;
    float var = 0.f;
#pragma unroll
    for (int j = 0; j < MAX_D / 32; ++j) {
        const int i = lane + 32 * j;
        if (i < d) var += (v[j] - mean) * (v[j] - mean);
    }
    var = warp_sum(var) / d;
    const float inv = 1.0f / sqrtf(var + LN_EPS);
#pragma unroll
    for (int j = 0; j < MAX_D / 32; ++j) {
        const int i = lane + 32 * j;
        if (i < d) {
            const float o = (v[j] - mean) * inv * g[i] + b[i];
            x[(size_t)r * d + i] = o;
            St<T>::st(xb + (size_t)r * d + i, o);
        }
    }
}

// Multi-query causal attention: CTA = (16 rows of one sequence, one head).
// K/V tiles of 64 positions are staged in shared memory and shared by the
// CTA's queries; each warp runs an online softmax for its queries.
template <typename T, int DH>
__global__ void __launch_bounds__(128) k_attention(AttArgs<T> a) {
    constexpr int QC = 16, KT = 64, OPL = (DH + 31) / 32;
    __shared__ float Ks[KT][DH + 1];
    __shared__ float Vs[KT][DH + 1];
    __shared__ float Qs[QC][DH];
    __shared__ int qpos[QC];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int h = blockIdx.y;
    const int seq = a.g0 / a.q_per_seq + blockIdx.z;
    const int r_lo = max(0, seq * a.q_per_seq - a.g0);
    const int r_hi = min(a.count, (seq + 1) * a.q_per_seq - a.g0);
    const int rb = r_lo + blockIdx.x * QC;
    const int re = min(rb + QC, r_hi);
    if (rb >= re) return;
    const int s = a.row_seq[rb];
    if (s < 0) return;  // rows of one sequence are all active or all inactive
    const int nq = re - rb;
    for (int i = tid; i < QC * DH; i += blockDim.x) {
        const int qi = i / DH, c = i % DH;
        Qs[qi][c] = qi < nq ? St<T>::ld(a.q + (size_t)(rb + qi) * a.d + h * DH + c) * a.scale : 0.f;
    }
    if (tid < QC) qpos[tid] = tid < nq ? a.row_pos[rb + tid] : -1;
    __syncthreads();
    const int maxpos = qpos[nq - 1];
    const size_t base = kv_index(a.kv, a.nh, DH, a.layer, s, h, 0);
    float m[4], l[4], o[4][OPL];
#pragma unroll
    for (int qq = 0; qq < 4; ++qq) {
        m[qq] = -INFINITY;
        l[qq] = 0.f;
#pragma unroll
        for (int c = 0; c < OPL; ++c) o[qq][c] = 0.f;
    }
    for (int k0 = 0; k0 <= maxpos; k0 += KT) {
        for (int i = tid; i < KT * DH; i += blockDim.x) {
            const int j = i / DH, c = i % DH;
            const bool ok = k0 + j <= maxpos;
            Ks[j][c] = ok ? St<T>::ld(a.kc + base + (size_t)(k0 + j) * DH + c) : 0.f;
            Vs[j][c] = ok ? St<T>::ld(a.vc + base + (size_t)(k0 + j) * DH + c) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
            const int qi = warp + 4 * qq;
            if (qi >= nq) break;
            const int qp = qpos[qi];
            float s0 = 0.f, s1 = 0.f;
#pragma unroll
            for (int c = 0; c < DH; ++c) {
                s0 = fmaf(Qs[qi][c], Ks[lane][c], s0);
                s1 = fmaf(Qs[qi][c], Ks[lane + 32][c], s1);
            }
            if (k0 + lane > qp) s0 = -INFINITY;
            if (k0 + lane + 32 > qp) s1 = -INFINITY;
            const float mt = warp_max(fmaxf(s0, s1));
            const float mn = fmaxf(m[qq], mt);
            const float corr = expf(m[qq] - mn);  // exp(-inf) = 0 on the first tile
            const float p0 = expf(s0 - mn), p1 = expf(s1 - mn);
            l[qq] = l[qq] * corr + warp_sum(p0 + p1);
#pragma unroll
            for (int c = 0; c < OPL; ++c) o[qq][c] *= corr;
            for (int jj = 0; jj < 32; ++jj) {
                const float pa = __shfl_sync(0xffffffffu, p0, jj);
                const float pb = __shfl_sync(0xffffffffu, p1, jj);
#pragma unroll
                for (int c = 0; c < OPL; ++c) {
                    const int cc = lane + 32 * c;
                    if (cc < DH) o[qq][c] = fmaf(pa, Vs[jj][cc], fmaf(pb, Vs[jj + 32][cc], o[qq][c]));
                }
            }
            m[qq] = mn;
        }
        __syncthreads();
    }
#pragma unroll
    for (int qq = 0; qq < 4; ++qq) {
        const int qi = warp + 4 * qq;
        if (qi >= nq) break;
        const float inv = 1.0f / (a.attnhp ? l[qq] + expf(-m[qq]) : l[qq]);
#pragma unroll
        for (int c = 0; c < OPL; ++c) {
            const int cc = lane + 32 * c;
            if (cc >= DH) continue;
            if (a.attnhp) {  // h <- h + tanh(a) (App. D.4)
                const size_t xi = (size_t)(rb + qi) * a.d + h * DH + cc;
                const float hn = a.x[xi] + tanhf(o[qq][c] * inv);
                a.x[xi] = hn;
                St<T>::st(a.hb + (size_t)(rb + qi) * 2 * a.d + a.d + h * DH + cc, hn);
            } else {
                St<T>::st(a.out + (size_t)(rb + qi) * a.d + h * DH + cc, o[qq][c] * inv);
            }
        }
    }
}

// ----------------------------------------------------------------------
// CTA-level pieces used by the single-position kernels (draft, AR, head)
// ----------------------------------------------------------------------

// y[o] = sum_i W[o][i] x[i] (+ b[o]) for o < out: one warp per output.
template <typename TW>
__device__ void cta_matvec(const TW* W, const float* bias, const float* x, int in, int out,
                           float* y) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    for (int o = warp; o < out; o += nw) {
        float acc = 0.f;
        const TW* row = W + (size_t)o * in;
        for (int i = lane; i < in; i += 32) acc = fmaf(St<TW>::ld(row + i), x[i], acc);
        acc = warp_sum(acc);
        if (lane == 0) y[o] = acc + (bias ? bias[o] : 0.f);
    }
}

__device__ void cta_layernorm(float* x, int d, const float* g, const float* b) {
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        float s = 0.f;
        for (int i = lane; i < d; i += 32) s += x[i];
        const float mean = warp_sum(s) / d;
        float v = 0.f;
        for (int i = lane; i < d; i += 32) v += (x[i] - mean) * (x[i] - mean);
        const float inv = 1.0f / sqrtf(warp_sum(v) / d + LN_EPS);
        for (int i = lane; i < d; i += 32) x[i] = (x[i] - mean) * inv * g[i] + b[i];
    }
}

// In-warp log-softmax of v[0..n).
__device__ void warp_log_softmax(float* v, int n) {
    const int lane = threadIdx.x & 31;
    float mx = -INFINITY;
    for (int i = lane; i < n; i += 32) mx = fmaxf(mx, v[i]);
    mx = warp_max(mx);
    float s = 0.f;
    for (int i = lane; i < n; i += 32) s += expf(v[i] - mx);
    const float lz = mx + logf(warp_sum(s));
    __syncwarp();
    for (int i = lane; i < n; i += 32) v[i] -= lz;
    __syncwarp();
}

// Head of Sec. 4.2 from h (shared memory, fp32): out = [log w | mu | s | log f].
// e and a are shared scratch of 3d and d floats.
__device__ void cta_head(const HeadW& hw, int d, int M, int K, const float* h, float* e, float* a,
                         float* out) {
    cta_matvec<float>(hw.E, nullptr, h, d, 3 * d, e);
    cta_matvec<float>(hw.v_k1, hw.b_k1, h, d, d, a);
    __syncthreads();
    cta_matvec<float>(hw.v_w, hw.b_w, e, d, M, out);
    cta_matvec<float>(hw.v_mu, hw.b_mu, e + d, d, M, out + M);
    cta_matvec<float>(hw.v_s, hw.b_s, e + 2 * d, d, M, out + 2 * M);
    for (int i = threadIdx.x; i < d; i += blockDim.x) a[i] = tanhf(a[i]);
    __syncthreads();
    cta_matvec<float>(hw.v_k2, hw.b_k2, a, d, K, out + 3 * M);
    __syncthreads();
    const int warp = threadIdx.x >> 5;
    if (warp == 0) warp_log_softmax(out, M);
    if (warp == 1) warp_log_softmax(out + 3 * M, K);
    __syncthreads();
}

// Online-softmax state merge (m, l, o) <- (m, l, o) (+) (m2, l2, o2).
template <int DH>
__device__ __forceinline__ void softmax_merge(float& m, float& l, float* o, float m2, float l2,
                                              const float* o2) {
    if (m2 == -INFINITY) return;
    if (m == -INFINITY) {
        m = m2; l = l2;
#pragma unroll
        for (int c = 0; c < DH; ++c) o[c] = o2[c];
        return;
    }
    const float mn = fmaxf(m, m2), a = expf(m - mn), b = expf(m2 - mn);
    l = l * a + l2 * b;
#pragma unroll
    for (int c = 0; c < DH; ++c) o[c] = o[c] * a + o2[c] * b;
    m = mn;
}

// One query per head over keys 0..n_keys-1 of one sequence and layer.
// Warp w takes head w % nh and the (w / nh)-th of nw/nh contiguous key
// ranges; lanes stride over keys with a lane-private online softmax, then
// warps merge through shared memory.  q: [nh*DH] fp32 (unscaled), out:
// [nh*DH].  scratch: nw * (DH + 2) floats.
template <typename T, int DH>
__device__ void cta_attend_one(const float* q, const T* kc, const T* vc, int n_keys, int nh,
                               int n_max, float scale, float* out, float* scratch, bool attnhp = false) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    const int h = warp % nh, split = warp / nh, S = nw / nh;
    const int per = (n_keys + S - 1) / S;
    const int lo = split * per, hi = min(n_keys, lo + per);
    float qr[DH];
#pragma unroll
    for (int c = 0; c < DH; ++c) qr[c] = q[h * DH + c] * scale;
    float m = -INFINITY, l = 0.f, o[DH];
#pragma unroll
    for (int c = 0; c < DH; ++c) o[c] = 0.f;
    const T* kb = kc + (size_t)h * n_max * DH;
    const T* vb = vc + (size_t)h * n_max * DH;
    for (int j = lo + lane; j < hi; j += 32) {
        float kr[DH];
        load_row<T>(kb + (size_t)j * DH, kr, DH);
        float sc = 0.f;
#pragma unroll
        for (int c = 0; c < DH; ++c) sc = fmaf(qr[c], kr[c], sc);
        const float mn = fmaxf(m, sc), corr = expf(m - mn), p = expf(sc - mn);
        l = l * corr + p;
        float vr[DH];
        load_row<T>(vb + (size_t)j * DH, vr, DH);
#pragma unroll
        for (int c = 0; c < DH; ++c) o[c] = fmaf(p, vr[c], o[c] * corr);
        m = mn;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
        const float l2 = __shfl_xor_sync(0xffffffffu, l, off);
        float o2[DH];
#pragma unroll
        for (int c = 0; c < DH; ++c) o2[c] = __shfl_xor_sync(0xffffffffu, o[c], off);
        softmax_merge<DH>(m, l, o, m2, l2, o2);
    }
    float* sw = scratch + warp * (DH + 2);
    if (lane == 0) {
        sw[0] = m;
        sw[1] = l;
#pragma unroll
        for (int c = 0; c < DH; ++c) sw[2 + c] = o[c];
    }
    __syncthreads();
    for (int t = threadIdx.x; t < nh * DH; t += blockDim.x) {
        const int hh = t / DH, c = t % DH;
        float mm = -INFINITY, ll = 0.f, oo = 0.f;
        for (int sp = 0; sp < S; ++sp) {
            const float* src = scratch + (sp * nh + hh) * (DH + 2);
            const float m2 = src[0];
            if (m2 == -INFINITY) continue;
            if (mm == -INFINITY) { mm = m2; ll = src[1]; oo = src[2 + c]; continue; }
            const float mn = fmaxf(mm, m2), a = expf(mm - mn), b = expf(m2 - mn);
            ll = ll * a + src[1] * b;
            oo = oo * a + src[2 + c] * b;
            mm = mn;
        }
        out[t] = attnhp ? oo / (ll + expf(-mm)) : oo / ll;
    }
    __syncthreads();
}

// Single-query attention for q_per_seq == 1 (autoregressive step): one CTA
// per row covering all heads.
template <typename T, int DH>
__global__ void __launch_bounds__(256) k_attention_single(AttArgs<T> a) {
    __shared__ float qs[MAX_D];
    __shared__ float os[MAX_D];
    __shared__ float scratch[8 * (64 + 2)];
    const int r = blockIdx.x;
    const int s = a.row_seq[r];
    if (s < 0) return;
    for (int i = threadIdx.x; i < a.d; i += blockDim.x) qs[i] = St<T>::ld(a.q + (size_t)r * a.d + i);
    __syncthreads();
    const size_t base = kv_index(a.kv, a.nh, DH, a.layer, s, 0, 0);
    cta_attend_one<T, DH>(qs, a.kc + base, a.vc + base, a.row_pos[r] + 1, a.nh, a.kv.n_max,
                          a.scale, os, scratch, a.attnhp != 0);
    for (int i = threadIdx.x; i < a.d; i += blockDim.x) {
        if (a.attnhp) {  // h <- h + tanh(a) (App. D.4)
            const float hn = a.x[(size_t)r * a.d + i] + tanhf(os[i]);
            a.x[(size_t)r * a.d + i] = hn;
            St<T>::st(a.hb + (size_t)r * 2 * a.d + a.d + i, hn);
        } else {
            St<T>::st(a.out + (size_t)r * a.d + i, os[i]);
        }
    }
}

// Head outputs from the batched pre-activations hd4 = [E h | V_k1 h + b_k1]
// (Sec. 4.2): w, mu, sigma logits from e1, e2, e3 and mark logits from
// tanh(.), then the two log-softmaxes.  One warp per row; the output maps
// (transposed, [d][3M+K]) are staged in shared memory when they fit.
// Small maps of the heads (Sec. 4.2) over 16 rows of hd4 = [E h | V_k1 h +
// b_k1] per CTA: out[o] = b[o] + sum_i act(o)[i] W_g[i][o], act = e_1, e_2,
// e_3 or tanh(V_k1 h + b_k1) by the output's group g (w logits, mu, log
// sigma, mark logits), then log-softmax of the w and the mark logits.  For
// each group in turn thread 0 copies the group's map (d x cnt, contiguous
// in head_out_g) and the 16 rows' inputs into shared memory by bulk copies
// (rows padded by 4 floats: the two rows a warp reads sit in distinct
// banks); thread t then takes row t / 16 and the group's outputs t % 16 +
// 16 j, j < NJ, so a row's sixteen threads are consecutive lanes and its
// log-softmax sums are four shuffles.
constexpr int HR_ROWS = 16;
__host__ __device__ inline size_t head_rows_smem(int d, int M, int K) {
    return sizeof(float) * ((size_t)HR_ROWS * (d + 4) + (size_t)d * (M > K ? M : K)) + 16;
}
// acc[j] += sum_i xr[i] wg[i][sub + 16 j] for j < J (J <= NJ, outputs < cnt).
template <int NJ, int J>
__device__ __forceinline__ void head_rows_dot(float (&acc)[NJ], const float* xr, const float* wg, int d, int cnt,
                                              int sub) {
    if constexpr (J <= NJ) {
#pragma unroll 4
        for (int i = 0; i < d; ++i) {
            const float xv = xr[i];
            const float* wr = wg + i * cnt + sub;
#pragma unroll
            for (int j = 0; j < J; ++j)
                if (sub + 16 * j < cnt) acc[j] = fmaf(wr[16 * j], xv, acc[j]);
        }
    }
}

template <int NJ>
__global__ void __launch_bounds__(256) k_head_rows(DevModel m, Work w, int count) {
    extern __shared__ __align__(16) float hsm[];
    const int d = m.d, M = m.M, K = m.K, WO = 3 * M + K, ld = d + 4;
    uint64_t* bar = (uint64_t*)hsm;
    float* xs = hsm + 4;                // [16][d + 4]
    float* wg = xs + HR_ROWS * ld;      // [d][cnt]: this group's map
    const int r0 = blockIdx.x * HR_ROWS, rows = min(HR_ROWS, count - r0);
    const int t = threadIdx.x, rr = t >> 4, sub = t & 15, r = r0 + rr;
    const bool live = r < count && w.row_seq[r] >= 0;
    float* dst = w.heads + (size_t)r * WO;
    const float* xr = xs + rr * ld;
    if (t == 0) {
        mbar_init(bar, 1);
        mbar_fence_init();
    }
    __syncthreads();
    int col0 = 0;
    bool ok = true;
    for (int g = 0; g < 4; ++g) {
        const int cnt = g < 3 ? M : K;
        if (t == 0) {  // the previous group's rows and map are consumed (barrier below)
            const uint32_t wbytes = (uint32_t)(d * cnt * 4), rbytes = (uint32_t)(d * 4);
            mbar_arrive_expect_tx(bar, wbytes + rbytes * rows);
            bulk_load(wg, m.head_out_g + (size_t)d * col0, wbytes, bar);
            for (int q = 0; q < rows; ++q) bulk_load(xs + q * ld, w.hd4 + (size_t)(r0 + q) * 4 * d + g * d, rbytes, bar);
        }
        ok = mbar_wait(bar, g & 1, w.err, 6) && ok;
        if (g == 3) {
            for (int idx = t; idx < rows * d; idx += 256) {
                const int q = idx / d, i = idx - q * d;
                xs[q * ld + i] = tanhf(xs[q * ld + i]);
            }
            __syncthreads();
        }
        float acc[NJ];
#pragma unroll
        for (int j = 0; j < NJ; ++j) acc[j] = 0.f;
        if (rr < rows) {
            // as many accumulators as the group needs (the mixture groups
            // are narrower than the mark group)
            const int nj = (cnt + 15) / 16;
            if (nj == 1) head_rows_dot<NJ, 1>(acc, xr, wg, d, cnt, sub);
            else if (nj == 2) head_rows_dot<NJ, 2>(acc, xr, wg, d, cnt, sub);
            else if (nj <= 4) head_rows_dot<NJ, 4>(acc, xr, wg, d, cnt, sub);
            else if (nj <= 8) head_rows_dot<NJ, 8>(acc, xr, wg, d, cnt, sub);
            else if (nj <= 16) head_rows_dot<NJ, 16>(acc, xr, wg, d, cnt, sub);
            else head_rows_dot<NJ, 32>(acc, xr, wg, d, cnt, sub);
        }
        float mx = -INFINITY;
#pragma unroll
        for (int j = 0; j < NJ; ++j)
            if (sub + 16 * j < cnt) {
                acc[j] += m.head_out_b[col0 + sub + 16 * j];
                mx = fmaxf(mx, acc[j]);
            }
        float lz = 0.f;
        if (g == 0 || g == 3) {  // log-softmax over the row's sixteen threads
#pragma unroll
            for (int o = 1; o < 16; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            float sm = 0.f;
#pragma unroll
            for (int j = 0; j < NJ; ++j)
                if (sub + 16 * j < cnt) sm += expf(acc[j] - mx);
#pragma unroll
            for (int o = 1; o < 16; o <<= 1) sm += __shfl_xor_sync(0xffffffffu, sm, o);
            lz = mx + logf(sm);
        }
        if (live && ok) {
#pragma unroll
            for (int j = 0; j < NJ; ++j)
                if (sub + 16 * j < cnt) dst[col0 + sub + 16 * j] = acc[j] - lz;
        }
        col0 += cnt;
        __syncthreads();  // every thread is done with this group's shared data
    }
}

static int head_rows_supported(const DevModel& m) {
    const int mk = m.M > m.K ? m.M : m.K;
    return m.d % 4 == 0 && mk <= 512 && head_rows_smem(m.d, m.M, m.K) <= 220 * 1024;
}

static cudaError_t launch_head_rows(const DevModel& m, const Work& w, int R, cudaStream_t st) {
    const int mk = m.M > m.K ? m.M : m.K, nj = (mk + 15) / 16;
    const size_t sm = head_rows_smem(m.d, m.M, m.K);
    const dim3 grid((R + HR_ROWS - 1) / HR_ROWS);
    auto go = [&](auto kern) {
        if (sm > 48 * 1024) {
            const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
            if (e != cudaSuccess) return e;
        }
        kern<<<grid, 256, sm, st>>>(m, w, R);
        return cudaGetLastError();
    };
    if (nj <= 1) return go(k_head_rows<1>);
    if (nj <= 2) return go(k_head_rows<2>);
    if (nj <= 4) return go(k_head_rows<4>);
    if (nj <= 8) return go(k_head_rows<8>);
    if (nj <= 16) return go(k_head_rows<16>);
    return go(k_head_rows<32>);
}

// x = hi + lo with hi = bf16(x), lo = bf16(x - hi), over n pairs of values.
__global__ void k_split_rows(const float* __restrict__ x, bf16* hi, bf16* lo, long long n) {
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        const float2 v = reinterpret_cast<const float2*>(x)[i];
        const __nv_bfloat162 h = __floats2bfloat162_rn(v.x, v.y);
        const float2 hf = __bfloat1622float2(h);
        reinterpret_cast<__nv_bfloat162*>(hi)[i] = h;
        reinterpret_cast<__nv_bfloat162*>(lo)[i] = __floats2bfloat162_rn(v.x - hf.x, v.y - hf.y);
    }
}

__global__ void __launch_bounds__(256) k_head_out(DevModel m, Work w, int count, int stage) {
    extern __shared__ float hsm[];
    const int d = m.d, M = m.M, K = m.K, WO = 3 * M + K;
    const float* Wt = m.head_out_t;
    if (stage) {
        for (int i = threadIdx.x; i < d * WO; i += blockDim.x) hsm[i] = Wt[i];
        Wt = hsm;
        __syncthreads();
    }
    float* xs = hsm + (stage ? d * WO : 0) + (threadIdx.x >> 5) * 4 * d;  // per-warp row copy
    const int lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    for (int r = blockIdx.x * nw + (threadIdx.x >> 5); r < count; r += gridDim.x * nw) {
        if (w.row_seq[r] < 0) continue;
        const float* src = w.hd4 + (size_t)r * 4 * d;
        for (int i = lane; i < 4 * d; i += 32) xs[i] = i < 3 * d ? src[i] : tanhf(src[i]);
        __syncwarp();
        float out[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int o = lane + 32 * j;
            out[j] = 0.f;
            if (o >= WO) continue;
            // which input block feeds output o: e1 (w), e2 (mu), e3 (sigma), tanh part (marks)
            const int part = o < M ? 0 : (o < 2 * M ? 1 : (o < 3 * M ? 2 : 3));
            const float* xin = xs + part * d;
            float acc = m.head_out_b[o];
            for (int i = 0; i < d; ++i) acc = fmaf(Wt[(size_t)i * WO + o], xin[i], acc);
            out[j] = acc;
        }
        // log-softmax over [0, M) and [3M, 3M+K)
        float mx_w = -INFINITY, mx_k = -INFINITY;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int o = lane + 32 * j;
            if (o < M) mx_w = fmaxf(mx_w, out[j]);
            else if (o >= 3 * M && o < WO) mx_k = fmaxf(mx_k, out[j]);
        }
        mx_w = warp_max(mx_w);
        mx_k = warp_max(mx_k);
        float sw = 0.f, sk = 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int o = lane + 32 * j;
            if (o < M) sw += expf(out[j] - mx_w);
            else if (o >= 3 * M && o < WO) sk += expf(out[j] - mx_k);
        }
        const float lzw = mx_w + logf(warp_sum(sw)), lzk = mx_k + logf(warp_sum(sk));
        float* dst = w.heads + (size_t)r * WO;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int o = lane + 32 * j;
            if (o < WO) dst[o] = o < M ? out[j] - lzw : (o >= 3 * M ? out[j] - lzk : out[j]);
        }
        __syncwarp();
    }
}

// ======================================================================
// draft: catch-up + gamma draft events, one CTA per sequence
// ======================================================================
struct DraftArgs {
    DevModel m;
    KVCache kv;
    SeqState ss;
    const CallParams* P;
    DevStats* st;
    float* heads;     // [Bmax][gamma_max][W]
    int gamma, gamma_max, stage, stage_bytes;
};

template <typename T>
__device__ const T* rebase(const void* p, const char* base, const char* nb) {
    return (const T*)(nb + ((const char*)p - base));
}

template <typename T, int DH>
__device__ void draft_encode(const DevModel& m, const DraftArgs& a, int s, int p, float* x,
                             float* xin, float* qkv, float* att, float* tmp, float* hid,
                             float* scratch) {
    const int d = m.d, F = m.F, tid = threadIdx.x, nt = blockDim.x;
    const SeqState& ss = a.ss;
    const size_t so = (size_t)s * ss.n_max + p;
    const double t = ss.t[so];
    const int k = ss.k[so];
    for (int i = tid; i < d / 2; i += nt) embed_pair(m, t, k, i, &x[2 * i], &x[2 * i + 1]);
    __syncthreads();
    T* kc = (T*)a.kv.k;
    T* vc = (T*)a.kv.v;
    const float scale = rsqrtf((float)DH);
    for (int l = 0; l < m.L; ++l) {
        const LayerW& L = m.layer[l];
        for (int i = tid; i < d; i += nt) xin[i] = St<T>::rnd(x[i]);
        __syncthreads();
        cta_matvec<T>((const T*)L.w_qkv, L.b_qkv, xin, d, 3 * d, qkv);
        __syncthreads();
        const size_t base = kv_index(a.kv, m.nh, DH, l, s, 0, 0);
        for (int i = tid; i < 3 * d; i += nt) {
            const float v = St<T>::rnd(qkv[i]);
            qkv[i] = v;
            if (i >= d) {
                const int which = i / d, cc = i - which * d, h = cc / DH, e = cc - h * DH;
                St<T>::st((which == 1 ? kc : vc) + base + ((size_t)h * a.kv.n_max + p) * DH + e, v);
            }
        }
        __syncthreads();
        cta_attend_one<T, DH>(qkv, kc + base, vc + base, p + 1, m.nh, a.kv.n_max, scale, att,
                              scratch);
        for (int i = tid; i < d; i += nt) att[i] = St<T>::rnd(att[i]);
        __syncthreads();
        cta_matvec<T>((const T*)L.w_o, L.b_o, att, d, d, tmp);
        __syncthreads();
        for (int i = tid; i < d; i += nt) x[i] += tmp[i];
        __syncthreads();
        cta_layernorm(x, d, L.ln1_g, L.ln1_b);
        __syncthreads();
        for (int i = tid; i < d; i += nt) xin[i] = St<T>::rnd(x[i]);
        __syncthreads();
        cta_matvec<T>((const T*)L.w_1, L.b_1, xin, d, F, hid);
        __syncthreads();
        for (int i = tid; i < F; i += nt) hid[i] = St<T>::rnd(fmaxf(hid[i], 0.f));
        __syncthreads();
        cta_matvec<T>((const T*)L.w_2, L.b_2, hid, F, d, tmp);
        __syncthreads();
        for (int i = tid; i < d; i += nt) x[i] += tmp[i];
        __syncthreads();
        cta_layernorm(x, d, L.ln2_g, L.ln2_b);
        __syncthreads();
    }
}

template <typename T, int DH>
__global__ void __launch_bounds__(128) k_draft(DraftArgs a) {
    extern __shared__ __align__(16) char smem[];
    const int s = blockIdx.x;
    const CallParams& P = *a.P;
    if (s >= P.B || a.ss.done[s]) return;
    DevModel m = a.m;
    if (a.stage) {
        // copy the whole model into shared memory and point at the copy
        const int4* src = (const int4*)m.base;
        int4* dst = (int4*)smem;
        for (size_t i = threadIdx.x; i < m.bytes / 16; i += blockDim.x) dst[i] = src[i];
        const char* nb = smem;
        m.type_emb = rebase<float>(m.type_emb, m.base, nb);
        m.tenc = rebase<double>(m.tenc, m.base, nb);
        for (int l = 0; l < m.L; ++l) {
            LayerW& L = m.layer[l];
            L.w_qkv = rebase<char>(L.w_qkv, m.base, nb); L.b_qkv = rebase<float>(L.b_qkv, m.base, nb);
            L.w_o = rebase<char>(L.w_o, m.base, nb);     L.b_o = rebase<float>(L.b_o, m.base, nb);
            L.ln1_g = rebase<float>(L.ln1_g, m.base, nb); L.ln1_b = rebase<float>(L.ln1_b, m.base, nb);
            L.w_1 = rebase<char>(L.w_1, m.base, nb);     L.b_1 = rebase<float>(L.b_1, m.base, nb);
            L.w_2 = rebase<char>(L.w_2, m.base, nb);     L.b_2 = rebase<float>(L.b_2, m.base, nb);
            L.ln2_g = rebase<float>(L.ln2_g, m.base, nb); L.ln2_b = rebase<float>(L.ln2_b, m.base, nb);
        }
        HeadW& H = m.head;
        H.E = rebase<float>(H.E, m.base, nb);
        H.v_w = rebase<float>(H.v_w, m.base, nb);   H.b_w = rebase<float>(H.b_w, m.base, nb);
        H.v_mu = rebase<float>(H.v_mu, m.base, nb); H.b_mu = rebase<float>(H.b_mu, m.base, nb);
        H.v_s = rebase<float>(H.v_s, m.base, nb);   H.b_s = rebase<float>(H.b_s, m.base, nb);
        H.v_k1 = rebase<float>(H.v_k1, m.base, nb); H.b_k1 = rebase<float>(H.b_k1, m.base, nb);
        H.v_k2 = rebase<float>(H.v_k2, m.base, nb); H.b_k2 = rebase<float>(H.b_k2, m.base, nb);
        __syncthreads();
    }
    const int d = m.d, F = m.F, M = m.M, K = m.K, W = m.head_width();
    float* x = (float*)(smem + a.stage_bytes);
    float* xin = x + d;
    float* qkv = xin + d;
    float* att = qkv + 3 * d;
    float* tmp = att + d;
    float* hid = tmp + d;
    float* e = hid + F;
    float* av = e + 3 * d;
    float* hd = av + d;
    float* scratch = hd + ((W + 3) & ~3);
    const SeqState& ss = a.ss;
    const int n = ss.n_emit[s];
    const int nd = ss.n_draft[s];
    for (int p = nd; p < n; ++p)
        draft_encode<T, DH>(m, a, s, p, x, xin, qkv, att, tmp, hid, scratch);
    if (threadIdx.x == 0) {
        // keys read per layer: positions 0..p for every encoded position p
        const long long last = n + a.gamma - 2;  // last encoded position
        const unsigned long long keys = (unsigned long long)((last + 1) * (last + 2) / 2 - (long long)nd * (nd + 1) / 2);
        atomicAdd(&a.st->draft_keys, keys);
    }
    for (int l = 1; l <= a.gamma; ++l) {
        const int p = n + l - 1;  // index of the drafted event
        cta_head(m.head, d, M, K, x, e, av, hd);
        float* rec = a.heads + ((size_t)s * a.gamma_max + (l - 1)) * W;
        for (int i = threadIdx.x; i < W; i += blockDim.x) rec[i] = hd[i];
        if (threadIdx.x == 0) {
            const U4 u = slot_uniforms(P.seed, (uint32_t)s, (uint32_t)p, 0u);
            const float tau = draw_tau(hd, M, u.x, u.y, u.z);
            const int k = pick_categorical_log(hd + 3 * M, K, u.w);
            const size_t o = (size_t)s * ss.n_max + p;
            ss.tau[o] = tau;
            ss.t[o] = ss.t[o - 1] + (double)tau;
            ss.k[o] = k;
        }
        __syncthreads();
        if (l < a.gamma) draft_encode<T, DH>(m, a, s, p, x, xin, qkv, att, tmp, hid, scratch);
    }
}

// ======================================================================
// verify epilogue: tests, first rejection, resampling, commit, rollback
// ======================================================================
struct EpiArgs {
    SeqState ss;
    const CallParams* P;
    const float* th;  // target heads, row s*(gamma+1)+l
    const float* dh;  // draft heads [Bmax][gamma_max][WD]
    int MT, MD, K, WT, WD, gamma, gamma_max;
    int poisson;  // draft = homogeneous Poisson process (App. D.3), parameters in *P
    DevStats* st;
};

// End-time stop rule (Alg. 1): a sequence with nn events is finished once
// N events are drawn or its last event lies beyond t_end.  Times increase
// along a sequence, so the events with t <= t_end are a prefix.
__device__ __forceinline__ bool seq_finished(const SeqState& ss, const CallParams& P, int s, int nn) {
    return nn >= P.H + P.N || (P.out_count && ss.t[(size_t)s * ss.n_max + nn - 1] > P.t_end);
}

// Number of generated events kept (t <= t_end, at most N) of a finished
// sequence; only the events of its last round can lie beyond t_end.
__device__ __forceinline__ int kept_count(const SeqState& ss, const CallParams& P, int s, int nn) {
    int c = min(nn - P.H, P.N);
    const double* t = ss.t + (size_t)s * ss.n_max + P.H;
    while (c > 0 && t[c - 1] > P.t_end) --c;
    return c;
}

__device__ void write_outputs(const SeqState& ss, const CallParams& P, int s, int n, int emitted) {
    const int lane = threadIdx.x & 31;
    for (int i = lane; i < emitted; i += 32) {
        const int p = n + i, j = p - P.H;
        if (j < P.N && (!P.out_count || ss.t[(size_t)s * ss.n_max + p] <= P.t_end)) {
            const size_t o = (size_t)s * ss.n_max + p, oo = (size_t)s * P.N + j;
            P.out_tau[oo] = ss.tau[o];
            P.out_t[oo] = ss.t[o];
            P.out_k[oo] = ss.k[o];
        }
    }
}

// One CTA (four warps) per sequence.  Warp 0: lane l-1 tests draft l (Sec.
// 4.3 "Verification"): accept tau iff u_tau < min(1, g_T/g_D), k iff u_k <
// min(1, f_T/f_D); L = first failing draft (ballot), gamma+1 if none.  At L
// the failing component(s) are redrawn: tau from g' by Theorem 1 (all 128
// threads: thread j takes iteration base+j, the smallest accepting index
// wins, which equals the sequential loop), k from f' (Eq. 4).  A full accept
// adds the bonus event from the target head after the last draft (unless
// NO_BONUS).
__global__ void __launch_bounds__(128) k_verify_epilogue(EpiArgs a) {
    pdl_wait();
    // per-component constants of both mixtures for the Theorem-1 loop
    __shared__ float cumT[MAX_MIX], muT[MAX_MIX], sgT[MAX_MIX], isT[MAX_MIX], cT[MAX_MIX];
    __shared__ float muD[MAX_MIX], isD[MAX_MIX], cD[MAX_MIX];
    __shared__ int sh_L, sh_at, sh_ak, sh_k;
    __shared__ float sh_umr, sh_tau;
    __shared__ int win_idx[4];
    __shared__ float win_tau[4];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int s = blockIdx.x;
    const CallParams& P = *a.P;
    const SeqState& ss = a.ss;
    if (s >= P.B || ss.done[s]) return;
    const int g = a.gamma, n = ss.n_emit[s];
    const size_t sb = (size_t)s * ss.n_max;
    if (warp == 0) {
        bool acc_t = true, acc_k = true;
        float tau_hat = 0.f, u_mr = 0.f;
        int k_hat = 0;
        if (lane < g) {
            const int p = n + lane;
            tau_hat = ss.tau[sb + p];
            k_hat = ss.k[sb + p];
            const float* hT = a.th + ((size_t)s * (g + 1) + lane) * a.WT;
            float lgD, lfD;
            if (a.poisson) {  // g_D = lambda exp(-lambda tau), f_D = p
                lgD = P.pois_log_rate - P.pois_rate * tau_hat;
                lfD = P.pois_logp[k_hat];
            } else {
                const float* hD = a.dh + ((size_t)s * a.gamma_max + lane) * a.WD;
                lgD = head_log_g(hD, a.MD, tau_hat);
                lfD = hD[3 * a.MD + k_hat];
            }
            const float rt = fminf(1.f, expf(head_log_g(hT, a.MT, tau_hat) - lgD));
            const float rk = fminf(1.f, expf(hT[3 * a.MT + k_hat] - lfD));
            const U4 u = slot_uniforms(P.seed, (uint32_t)s, (uint32_t)p, 1u);
            acc_t = u.x < rt;
            acc_k = u.y < rk;
            u_mr = u.z;
            if (P.trace)  // signed margins of the two tests (negative: accepted)
                P.trace[sb + p] = make_float4(u.x - rt, u.y - rk, 0.f, (float)a.st->loop_iters);
        }
        const unsigned fail = __ballot_sync(0xffffffffu, lane < g && !(acc_t && acc_k));
        const int L = fail ? __ffs(fail) : g + 1;  // 1-based
        if (P.trace && lane < g && lane < L) {
            // decision codes: 1 accepted draft, 2 time redrawn (Theorem 1),
            // 4 mark redrawn (Eq. 4); the first rejection may carry both
            const int code = lane < L - 1 ? 1 : (acc_t ? 0 : 2) | (acc_k ? 0 : 4);
            P.trace[sb + n + lane].z = (float)code;
        }
        const int src = L <= g ? L - 1 : 0;
        const bool at = __shfl_sync(0xffffffffu, acc_t, src);
        const bool ak = __shfl_sync(0xffffffffu, acc_k, src);
        const float umr = __shfl_sync(0xffffffffu, u_mr, src);
        const float tau = __shfl_sync(0xffffffffu, tau_hat, src);
        const int k = __shfl_sync(0xffffffffu, k_hat, src);
        if (L <= g && !at) {
            // constants of the time resampler: running sums of w_T (the
            // component pick), mu, sigma, 1/sigma and log w - log sigma.  The
            // log tau and log(2 pi)/2 terms of log g_T and log g_D cancel in
            // their difference.
            const float* hT = a.th + ((size_t)s * (g + 1) + src) * a.WT;
            const int MT = a.MT, MD = a.MD;
            for (int m = lane; m < MT; m += 32) {
                muT[m] = hT[MT + m];
                sgT[m] = expf(hT[2 * MT + m]);
                isT[m] = expf(-hT[2 * MT + m]);
                cT[m] = hT[m] - hT[2 * MT + m];
            }
            if (!a.poisson) {
                const float* hD = a.dh + ((size_t)s * a.gamma_max + src) * a.WD;
                for (int m = lane; m < MD; m += 32) {
                    muD[m] = hD[MD + m];
                    isD[m] = expf(-hD[2 * MD + m]);
                    cD[m] = hD[m] - hD[2 * MD + m];
                }
            }
            if (lane == 0) {
                float run = 0.f;
                for (int m = 0; m < MT; ++m) { run += expf(hT[m]); cumT[m] = run; }
            }
        }
        if (lane == 0) {
            sh_L = L;
            sh_at = at;
            sh_ak = ak;
            sh_umr = umr;
            sh_tau = tau;
            sh_k = k;
        }
    }
    __syncthreads();
    const int L = sh_L, A = L - 1;
    float tau = sh_tau;
    unsigned long long iters = 0, cap = 0;
    if (L <= g && !sh_at) {
        // Theorem 1: proposals from g_T, accepted with max(0, 1 - g_D / g_T)
        const int p = n + L - 1, MT = a.MT, MD = a.MD;
        const float totT = cumT[MT - 1];
        bool found = false;
        float last = 0.f;
        const int rcap = P.resample_cap;
        for (int base = 0; base < rcap && !found; base += 128) {
            const int it = base + tid;
            const bool live_it = it < rcap;
            const U4 u = slot_uniforms(P.seed, (uint32_t)s, (uint32_t)p, 2u + (uint32_t)it);
            const float target = u.x * totT;
            int z = MT - 1;
            for (int m = 0; m < MT; ++m)
                if (cumT[m] >= target) { z = m; break; }
            const float eps = sqrtf(-2.0f * logf(u.y)) * cospif(2.0f * u.z);
            const float lt = fmaf(sgT[z], eps, muT[z]);
            float mT = -INFINITY;
            for (int m = 0; m < MT; ++m) {
                const float q = (lt - muT[m]) * isT[m];
                mT = fmaxf(mT, cT[m] - 0.5f * q * q);
            }
            float sT = 0.f;
            for (int m = 0; m < MT; ++m) {
                const float q = (lt - muT[m]) * isT[m];
                sT += expf(cT[m] - 0.5f * q * q - mT);
            }
            const float tp = expf(lt);
            float ldiff;  // log g_D - log g_T at the proposal
            if (a.poisson) {
                const float HALF_LOG_2PI = 0.91893853320467274178f;
                ldiff = (P.pois_log_rate - P.pois_rate * tp) - (mT + logf(sT) - lt - HALF_LOG_2PI);
            } else {
                float mD = -INFINITY;
                for (int m = 0; m < MD; ++m) {
                    const float q = (lt - muD[m]) * isD[m];
                    mD = fmaxf(mD, cD[m] - 0.5f * q * q);
                }
                float sD = 0.f;
                for (int m = 0; m < MD; ++m) {
                    const float q = (lt - muD[m]) * isD[m];
                    sD += expf(cD[m] - 0.5f * q * q - mD);
                }
                ldiff = (mD + logf(sD)) - (mT + logf(sT));
            }
            const float al = fmaxf(0.f, 1.f - expf(ldiff));
            const unsigned okb = __ballot_sync(0xffffffffu, live_it && u.w < al);
            if (lane == 0) {
                win_idx[warp] = okb ? 32 * warp + __ffs(okb) - 1 : 1 << 30;
            }
            if (okb && lane == __ffs(okb) - 1) win_tau[warp] = tp;
            if (it == rcap - 1) last = tp;
            __syncthreads();
            int best = 1 << 30, bw = 0;
            for (int w = 0; w < 4; ++w)
                if (win_idx[w] < best) { best = win_idx[w]; bw = w; }
            if (best < (1 << 30)) {
                tau = win_tau[bw];
                iters = (unsigned long long)(base + best + 1);
                found = true;
            }
            __syncthreads();  // the winner slots are rewritten by the next step
        }
        if (!found) {  // the last proposal of the capped loop (iteration rcap - 1)
            if (tid == (rcap - 1) % 128) sh_tau = last;
            __syncthreads();
            tau = sh_tau;
            iters = (unsigned long long)rcap;
            cap = 1;
        }
    }
    if (warp != 0) return;
    int emitted;
    if (L <= g) {
        const int p = n + L - 1, src = L - 1;
        int k = sh_k;
        const float* hT = a.th + ((size_t)s * (g + 1) + src) * a.WT;
        // log f_D: the draft head's mark block, or log p of the Poisson draft
        const float* lfD = a.poisson ? P.pois_logp : a.dh + ((size_t)s * a.gamma_max + src) * a.WD + 3 * a.MD;
        if (!sh_ak && lane == 0) {
            // f' = norm(max(0, f_T - f_D)); zero mass -> draw from f_T
            const float umr = sh_umr;
            float tot = 0.f;
            for (int kk = 0; kk < a.K; ++kk) tot += fmaxf(0.f, expf(hT[3 * a.MT + kk]) - expf(lfD[kk]));
            if (tot < 1e-12f) {
                k = pick_categorical_log(hT + 3 * a.MT, a.K, umr);
            } else {
                const float target = umr * tot;
                float run = 0.f;
                k = a.K - 1;
                for (int kk = 0; kk < a.K; ++kk) {
                    run += fmaxf(0.f, expf(hT[3 * a.MT + kk]) - expf(lfD[kk]));
                    if (run >= target) { k = kk; break; }
                }
            }
        }
        k = __shfl_sync(0xffffffffu, k, 0);
        if (lane == 0) {
            ss.tau[sb + p] = tau;
            ss.t[sb + p] = ss.t[sb + p - 1] + (double)tau;
            ss.k[sb + p] = k;
        }
        emitted = L;
    } else if (!(P.flags & FLAG_NO_BONUS)) {
        const int p = n + g;
        if (lane == 0) {
            const float* hT = a.th + ((size_t)s * (g + 1) + g) * a.WT;
            const U4 u = slot_uniforms(P.seed, (uint32_t)s, (uint32_t)p, 0u);
            if (P.trace)  // 8: bonus event from the target head after the last draft
                P.trace[sb + p] = make_float4(NAN, NAN, 8.f, (float)a.st->loop_iters);
            const float tb = draw_tau(hT, a.MT, u.x, u.y, u.z);
            ss.tau[sb + p] = tb;
            ss.t[sb + p] = ss.t[sb + p - 1] + (double)tb;
            ss.k[sb + p] = pick_categorical_log(hT + 3 * a.MT, a.K, u.w);
        }
        emitted = g + 1;
    } else {
        emitted = g;
    }
    __syncwarp();
    write_outputs(ss, P, s, n, emitted);
    if (lane == 0) {
        const int nn = n + emitted;
        ss.n_emit[s] = nn;
        ss.n_draft[s] = n + min(g - 1, A);
        const bool fin = seq_finished(ss, P, s, nn);
        ss.done[s] = fin;
        if (fin && P.out_count) P.out_count[s] = kept_count(ss, P, s, nn);
        atomicAdd(&a.st->rounds, 1ull);
        atomicAdd(&a.st->target_keys, (unsigned long long)(n + g));  // positions 0..n+g-1
        atomicAdd(&a.st->drafted, (unsigned long long)g);
        atomicAdd(&a.st->accepted, (unsigned long long)A);
        atomicAdd(&a.st->emitted, (unsigned long long)emitted);
        if (iters) atomicAdd(&a.st->resample_iters, iters);
        if (cap) atomicAdd(&a.st->cap_hits, cap);
    }
    pdl_trigger();
}

// Poisson draft (App. D.3): the gamma drafts of an active sequence, all at
// once since the draft ignores the history.  Position p = n + l uses its
// block-0 slot: tau = -log(u_comp) / lambda (inversion of the exponential
// CDF), mark from p with u_mark.  One thread per sequence keeps the
// absolute times a sequential fp64 sum.
__global__ void k_poisson_draft(SeqState ss, const CallParams* Pp, int gamma, int K) {
    pdl_wait();
    const int s = blockIdx.x * blockDim.x + threadIdx.x;
    const CallParams& P = *Pp;
    if (s < P.B && !ss.done[s]) {
        const int n = ss.n_emit[s];
        const size_t sb = (size_t)s * ss.n_max;
        double t = ss.t[sb + n - 1];
        for (int l = 0; l < gamma; ++l) {
            const int p = n + l;
            const U4 u = slot_uniforms(P.seed, (uint32_t)s, (uint32_t)p, 0u);
            const float tau = -logf(u.x) / P.pois_rate;
            t += (double)tau;
            ss.tau[sb + p] = tau;
            ss.t[sb + p] = t;
            ss.k[sb + p] = pick_categorical_log(P.pois_logp, K, u.w);
        }
    }
    pdl_trigger();
}

// Autoregressive sample (Sec. 4.2): one thread per sequence, head row s.
__global__ void k_ar_sample(SeqState ss, const CallParams* Pp, const float* heads, int M, int K,
                            int W, DevStats* st) {
    pdl_wait();
    const int s = blockIdx.x * blockDim.x + threadIdx.x;
    const CallParams& P = *Pp;
    if (s >= P.B || ss.done[s]) return;
    const int n = ss.n_emit[s];
    const float* hd = heads + (size_t)s * W;
    const U4 u = slot_uniforms(P.seed, (uint32_t)s, (uint32_t)n, 0u);
    const float tau = draw_tau(hd, M, u.x, u.y, u.z);
    const int k = pick_categorical_log(hd + 3 * M, K, u.w);
    const size_t o = (size_t)s * ss.n_max + n;
    ss.tau[o] = tau;
    ss.t[o] = ss.t[o - 1] + (double)tau;
    ss.k[o] = k;
    const int j = n - P.H;
    if (j < P.N && (!P.out_count || ss.t[o] <= P.t_end)) {
        const size_t oo = (size_t)s * P.N + j;
        P.out_tau[oo] = tau;
        P.out_t[oo] = ss.t[o];
        P.out_k[oo] = k;
    }
    ss.n_emit[s] = n + 1;
    const bool fin = seq_finished(ss, P, s, n + 1);
    ss.done[s] = fin;
    if (fin && P.out_count) P.out_count[s] = kept_count(ss, P, s, n + 1);
    atomicAdd(&st->rounds, 1ull);
    atomicAdd(&st->emitted, 1ull);
    atomicAdd(&st->target_keys, (unsigned long long)n);  // positions 0..n-1
    pdl_trigger();
}

// ======================================================================
// call set-up, round control, history, scoring
// ======================================================================
__global__ void k_begin(CallParams p, CallParams* dp, SeqState ss, DevStats* st) {
    const int s = blockIdx.x * blockDim.x + threadIdx.x;
    if (s == 0) {
        *dp = p;
        st->rounds = st->drafted = st->accepted = st->emitted = 0;
        st->resample_iters = st->cap_hits = st->loop_iters = 0;
        st->target_keys = st->draft_keys = 0;
        st->round_limit_hit = 0;
    }
    if (s < p.B) {
        ss.n_emit[s] = p.H;
        ss.n_draft[s] = p.H - 1;
        // a history that already ends beyond t_end generates nothing
        ss.done[s] = p.N <= 0 || (p.out_count && ss.t[(size_t)s * ss.n_max + p.H - 1] > p.t_end);
        if (p.out_count) p.out_count[s] = 0;
    }
}

// Any sequence still active?  Sets the WHILE condition of the round graph
// (or writes the flag for the host-driven loop).  Also enforces the
// round-count safety cap.
__global__ void __launch_bounds__(256) k_round_control(SeqState ss, const CallParams* Pp,
                                                       DevStats* st, cudaGraphConditionalHandle h,
                                                       int use_cond, int* active_out) {
    pdl_wait();
    __shared__ int cnt;
    if (threadIdx.x == 0) cnt = 0;
    __syncthreads();
    int c = 0;
    for (int s = threadIdx.x; s < Pp->B; s += blockDim.x) c += ss.done[s] == 0;
    if (c) atomicAdd(&cnt, c);
    __syncthreads();
    if (threadIdx.x == 0) {
        const unsigned long long it = ++st->loop_iters;
        int cont = cnt > 0;
        if (cont && it >= (unsigned long long)Pp->max_loops) {
            st->round_limit_hit = 1;
            cont = 0;
        }
        if (use_cond) cudaGraphSetConditional(h, cont ? 1u : 0u);
        if (active_out) *active_out = cont;
    }
}

__global__ void k_history_times(SeqState ss, int B, int H) {
    const int s = blockIdx.x * blockDim.x + threadIdx.x;
    if (s >= B) return;
    double t = 0.0;  // t_0 = 0; t_i = t_{i-1} + tau_i
    for (int p = 0; p < H; ++p) {
        const size_t o = (size_t)s * ss.n_max + p;
        t += (double)ss.tau[o];
        ss.t[o] = t;
    }
}

// Teacher-forced outputs of a span pass over q positions per sequence (q =
// len-1, or len when the head after the last event is wanted too): row r
// <-> (s, l), head predicts event l+1 (Eq. 2 terms log g(tau_{l+1}),
// log f(k_{l+1})).
__global__ void k_score_logs(SeqState ss, Work w, int M, int K, int len, int q, int g0, int rows,
                             float* out_heads, float* out_logg, float* out_logf) {
    const int r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r >= rows) return;
    const int W = 3 * M + K;
    const long long g = g0 + (long long)r;
    const int s = (int)(g / q), l = (int)(g % q);
    const float* hd = w.heads + (size_t)r * W;
    if (out_heads)
        for (int i = 0; i < W; ++i) out_heads[((size_t)s * len + l) * W + i] = hd[i];
    if (l + 1 >= len) return;
    const size_t o = (size_t)s * ss.n_max + l + 1;
    if (out_logg) out_logg[(size_t)s * len + l + 1] = head_log_g(hd, M, ss.tau[o]);
    if (out_logf) out_logf[(size_t)s * len + l + 1] = hd[3 * M + ss.k[o]];
    if (l == 0) {
        if (out_logg) out_logg[(size_t)s * len] = NAN;
        if (out_logf) out_logf[(size_t)s * len] = NAN;
    }
}

// log of the upper tail of the standard normal, 1 - Phi(z): for z > 0 from
// the scaled complementary error function, erfc(x) = erfcx(x) exp(-x^2),
// which stays finite far into the tail; for z <= 0 erfc itself (in [1, 2]).
__device__ __forceinline__ double log_normal_upper(double z) {
    const double x = z * 0.70710678118654752440;  // z / sqrt(2)
    return z > 0.0 ? log(0.5 * erfcx(x)) - x * x : log(0.5 * erfc(x));
}

// Survival term of the log-likelihood on [0, t_end] (Eq. 2): with the head
// after the last event (row of position len-1), log S(u) = log sum_m w_m
// (1 - Phi((log u - mu_m) / sigma_m)) at u = t_end - t_last, in fp64; 0 for
// u <= 0 (the window ends at or before the last event).
__global__ void k_score_survival(SeqState ss, Work w, int M, int K, int len, int g0, int rows, double t_end,
                                 double* out_logS) {
    const int r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r >= rows) return;
    const long long g = g0 + (long long)r;
    const int s = (int)(g / len), l = (int)(g % len);
    if (l != len - 1) return;
    const double u = t_end - ss.t[(size_t)s * ss.n_max + l];
    if (!(u > 0.0)) {
        out_logS[s] = 0.0;
        return;
    }
    const float* hd = w.heads + (size_t)r * (3 * M + K);
    const double lu = log(u);
    double mx = -INFINITY, acc = 0.0;
    for (int m = 0; m < M; ++m) {  // online log-sum-exp over the components
        const double v = (double)hd[m] + log_normal_upper((lu - (double)hd[M + m]) * exp(-(double)hd[2 * M + m]));
        if (v > mx) {
            acc = acc * exp(mx - v) + 1.0;
            mx = v;
        } else {
            acc += exp(v - mx);
        }
    }
    out_logS[s] = mx + log(acc);
}

// ======================================================================
// host launchers
// ======================================================================
#define DISPATCH_DH(DHV, ...)                                          \
    switch (DHV) {                                                     \
        case 8: { constexpr int DH = 8; __VA_ARGS__; } break;          \
        case 16: { constexpr int DH = 16; __VA_ARGS__; } break;        \
        case 32: { constexpr int DH = 32; __VA_ARGS__; } break;        \
        case 64: { constexpr int DH = 64; __VA_ARGS__; } break;        \
        default: return cudaErrorInvalidValue;                         \
    }

// Attention of one layer: bf16 caches use the bulk-copy / mma kernel of
// attn.cu; fp32 caches (the fp32 models) use the SIMT kernels above.
template <typename T>
static cudaError_t attention_launch(const AttArgs<T>& aa, const DevModel& m, const RowSpec& rs, int R,
                                    int nseg, const Work& w, cudaStream_t st) {
    if constexpr (sizeof(T) == 2) {
        // tcgen05 form (attn_tc.cu); TPPSD_ATTN_MMA=1 selects the mma.sync form
        if (m.attn_tc) return launch_attn_tc(aa, m.dh, m.nh, nseg, rs.mode == ROWS_STEP, w.attn, w.err, st);
        if (m.dh >= 16) return launch_attn_mma(aa, m.dh, m.nh, nseg, w.err, st);
    }
    if (rs.q == 1) {
        DISPATCH_DH(m.dh, (k_attention_single<T, DH><<<R, 256, 0, st>>>(aa)));
    } else {
        const dim3 ag((rs.q + 15) / 16, m.nh, nseg);
        DISPATCH_DH(m.dh, (k_attention<T, DH><<<ag, 128, 0, st>>>(aa)));
    }
    return cudaGetLastError();
}

template <typename T>
static cudaError_t forward_t(const DevModel& m, const KVCache& kv, const SeqState& ss,
                             const Work& w, const RowSpec& rs, bool want_heads, cudaStream_t st,
                             int* launches, const Prof* prof, const TcPlan* tc) {
    const int R = rs.count, d = m.d, F = m.F;
    if (R <= 0) return cudaSuccess;
    int nl = 0;
    if (!rs.pre_embedded) {
        const long long total = (long long)R * (d / 2);
        const long long want = (total + 255) / 256;
        const int blocks = (int)(want < 152 * 16 ? want : 152 * 16);
        PROF_MARK(prof, KC_EMBED, 1, st);
        if (const cudaError_t e = launch_k(k_embed<T>, dim3(blocks), dim3(256), 0, st, m, ss, rs, w)) return e;
        PROF_MARK(prof, KC_EMBED, 0, st);
        ++nl;
    }
    T* xb = (T*)w.xb;
    T* q = (T*)w.q;
    T* att = (T*)w.att;
    T* hid = (T*)w.hid;
    const dim3 blk(256);
    auto grid = [&](int N) { return dim3((N + 63) / 64, (R + 63) / 64); };
    const int nseg = (int)((rs.g0 + (long long)R - 1) / rs.q - rs.g0 / rs.q + 1);
    const bool use_tc = tc && tc->enabled && m.dtype == 1;
    for (int l = 0; l < m.L && m.enc == 2; ++l) {
        // AttNHP layer (App. D.4): q, k, v = W [z; h] + b from the [z | h] rows
        // (K/V into the cache), then attention with the 1 + sum f normaliser
        // whose epilogue applies h <- h + tanh(a)
        const LayerW& L = m.layer[l];
        cudaError_t e = cudaSuccess;
        PROF_MARK(prof, KC_GEMM_QKV, 1, st);
        if (use_tc) {
            TcGemmArgs g{};
            g.R = R; g.N = 3 * d; g.K = 2 * d; g.epi = EPI_TC_QKV; g.bias = L.b_qkv;
            g.q_out = (bf16*)q; g.kc = (bf16*)kv.k; g.vc = (bf16*)kv.v;
            g.row_seq = w.row_seq; g.row_pos = w.row_pos;
            g.d = d; g.nh = m.nh; g.dh = m.dh; g.layer = l; g.Bmax = kv.Bmax; g.n_max = kv.n_max;
            g.err = tc->err;
            g.v_f16 = m.v_f16;
            e = launch_gemm_tc(tc->a_zh, tc->layer[l].wqkv, g, tc->bn_qkv, st);
        } else {
            GemmArgs<T> g{};
            g.A = xb; g.W = (const T*)L.w_qkv; g.bias = L.b_qkv; g.R = R; g.N = 3 * d; g.K = 2 * d;
            g.q_out = q; g.kc = (T*)kv.k; g.vc = (T*)kv.v; g.row_seq = w.row_seq; g.row_pos = w.row_pos;
            g.d = d; g.nh = m.nh; g.dh = m.dh; g.layer = l; g.Bmax = kv.Bmax; g.n_max = kv.n_max;
            g.v_f16 = m.v_f16;
            k_gemm<T, EPI_QKV><<<grid(3 * d), blk, 0, st>>>(g);
            e = cudaGetLastError();
        }
        if (e != cudaSuccess) return e;
        PROF_MARK(prof, KC_GEMM_QKV, 0, st);
        AttArgs<T> aa{};
        aa.q = q; aa.kc = (const T*)kv.k; aa.vc = (const T*)kv.v; aa.out = att;
        aa.row_seq = w.row_seq; aa.row_pos = w.row_pos; aa.count = R; aa.q_per_seq = rs.q;
        aa.g0 = rs.g0; aa.d = d; aa.nh = m.nh; aa.layer = l; aa.kv = kv;
        aa.scale = 1.0f / sqrtf((float)m.dh);
        aa.attnhp = 1; aa.x = w.x; aa.hb = xb;
        PROF_MARK(prof, KC_ATTENTION, 1, st);
        if ((e = attention_launch<T>(aa, m, rs, R, nseg, w, st)) != cudaSuccess) return e;
        PROF_MARK(prof, KC_ATTENTION, 0, st);
        nl += 2;
    }
    // the fused block of layer l computes layer l + 1's Q, K, V (folded QKV)
    const bool fold = use_tc && tc->mlp && tc->mlp_cl && tc->qkv_fold;
    for (int l = 0; l < m.L && m.enc != 2; ++l) {
        const LayerW& L = m.layer[l];
        if (use_tc) {
            cudaError_t e;
            if (!(fold && l > 0)) {
                TcGemmArgs g{};
                g.R = R; g.N = 3 * d; g.K = d; g.epi = EPI_TC_QKV; g.bias = L.b_qkv;
                g.q_out = (bf16*)q; g.kc = (bf16*)kv.k; g.vc = (bf16*)kv.v;
                g.row_seq = w.row_seq; g.row_pos = w.row_pos;
                g.d = d; g.nh = m.nh; g.dh = m.dh; g.layer = l; g.Bmax = kv.Bmax; g.n_max = kv.n_max;
                g.err = tc->err;
                g.stall = tc->stall;
                g.v_f16 = m.v_f16;
                PROF_MARK(prof, KC_GEMM_QKV, 1, st);
                if ((e = launch_gemm_tc(tc->a_xb, tc->layer[l].wqkv, g, tc->bn_qkv, st)) != cudaSuccess) return e;
                PROF_MARK(prof, KC_GEMM_QKV, 0, st);
                ++nl;
            }
            AttArgs<T> aa{};
            aa.q = q; aa.kc = (const T*)kv.k; aa.vc = (const T*)kv.v; aa.out = att;
            aa.row_seq = w.row_seq; aa.row_pos = w.row_pos; aa.count = R; aa.q_per_seq = rs.q;
            aa.g0 = rs.g0; aa.d = d; aa.nh = m.nh; aa.layer = l; aa.kv = kv;
            aa.scale = 1.0f / sqrtf((float)m.dh);
            PROF_MARK(prof, KC_ATTENTION, 1, st);
            if ((e = attention_launch<T>(aa, m, rs, R, nseg, w, st)) != cudaSuccess) return e;
            PROF_MARK(prof, KC_ATTENTION, 0, st);
            if (tc->mlp) {
                MlpArgs ma{};
                ma.R = R; ma.F = F; ma.b_o = L.b_o; ma.ln1_g = L.ln1_g; ma.ln1_b = L.ln1_b;
                ma.b_1 = L.b_1; ma.b_2 = L.b_2; ma.ln2_g = L.ln2_g; ma.ln2_b = L.ln2_b;
                ma.x = w.x; ma.xb = (bf16*)xb; ma.err = tc->err;
                const int ln = l + 1 < m.L ? l + 1 : l;  // the layer whose Q, K, V are folded in
                if (fold && l + 1 < m.L) {
                    ma.qkv = 1; ma.b_qkv = m.layer[ln].b_qkv;
                    ma.q_out = (bf16*)q; ma.kc = (bf16*)kv.k; ma.vc = (bf16*)kv.v;
                    ma.row_seq = w.row_seq; ma.row_pos = w.row_pos;
                    ma.nh = m.nh; ma.dh = m.dh; ma.layer = ln; ma.Bmax = kv.Bmax; ma.n_max = kv.n_max;
                    ma.v_f16 = m.v_f16;
                }
                PROF_MARK(prof, KC_GEMM_FFN2, 1, st);
                e = tc->mlp_cl ? launch_mlp_cl(tc->a_att, tc->layer[l].wo_m, tc->layer[l].w1_m, tc->layer[l].w2_m,
                                               ma.qkv ? tc->layer[ln].wqkv_f : tc->layer[l].w2_m, ma, st)
                               : launch_mlp_tc(tc->a_att, tc->layer[l].wo_m, tc->layer[l].w1_m, tc->layer[l].w2_m, ma, st);
                if (e != cudaSuccess) return e;
                PROF_MARK(prof, KC_GEMM_FFN2, 0, st);
                nl += 2;
                continue;
            }
            TcGemmArgs go{};
            go.R = R; go.N = d; go.K = d; go.epi = EPI_TC_RESID_LN; go.bias = L.b_o;
            go.resid = w.x; go.x_out = w.x; go.xb_out = (bf16*)xb; go.ln_g = L.ln1_g; go.ln_b = L.ln1_b;
            go.err = tc->err;
            PROF_MARK(prof, KC_GEMM_O, 1, st);
            e = launch_gemm_ln_cluster(tc->a_att, tc->layer[l].wo, go, st);
            if (e != cudaSuccess) return e;
            PROF_MARK(prof, KC_GEMM_O, 0, st);
            TcGemmArgs g1{};
            g1.R = R; g1.N = F; g1.K = d; g1.epi = EPI_TC_RELU; g1.bias = L.b_1; g1.out_t = (bf16*)hid;
            g1.err = tc->err;
            PROF_MARK(prof, KC_GEMM_FFN1, 1, st);
            if ((e = launch_gemm_tc(tc->a_xb, tc->layer[l].w1, g1, tc->bn_ffn1, st)) != cudaSuccess) return e;
            PROF_MARK(prof, KC_GEMM_FFN1, 0, st);
            TcGemmArgs g2{};
            g2.R = R; g2.N = d; g2.K = F; g2.epi = EPI_TC_RESID_LN; g2.bias = L.b_2;
            g2.resid = w.x; g2.x_out = w.x; g2.xb_out = (bf16*)xb; g2.ln_g = L.ln2_g; g2.ln_b = L.ln2_b;
            g2.err = tc->err;
            PROF_MARK(prof, KC_GEMM_FFN2, 1, st);
            e = launch_gemm_ln_cluster(tc->a_hid, tc->layer[l].w2, g2, st);
            if (e != cudaSuccess) return e;
            PROF_MARK(prof, KC_GEMM_FFN2, 0, st);
            nl += 4;
            continue;
        }
        GemmArgs<T> g{};
        g.A = xb; g.W = (const T*)L.w_qkv; g.bias = L.b_qkv; g.R = R; g.N = 3 * d; g.K = d;
        g.q_out = q; g.kc = (T*)kv.k; g.vc = (T*)kv.v; g.row_seq = w.row_seq; g.row_pos = w.row_pos;
        g.d = d; g.nh = m.nh; g.dh = m.dh; g.layer = l; g.Bmax = kv.Bmax; g.n_max = kv.n_max;
        g.v_f16 = m.v_f16;
        PROF_MARK(prof, KC_GEMM_QKV, 1, st);
        k_gemm<T, EPI_QKV><<<grid(3 * d), blk, 0, st>>>(g);
        PROF_MARK(prof, KC_GEMM_QKV, 0, st);
        AttArgs<T> aa{};
        aa.q = q; aa.kc = (const T*)kv.k; aa.vc = (const T*)kv.v; aa.out = att;
        aa.row_seq = w.row_seq; aa.row_pos = w.row_pos; aa.count = R; aa.q_per_seq = rs.q;
        aa.g0 = rs.g0; aa.d = d; aa.nh = m.nh; aa.layer = l; aa.kv = kv;
        aa.scale = 1.0f / sqrtf((float)m.dh);
        PROF_MARK(prof, KC_ATTENTION, 1, st);
        {
            const cudaError_t e = attention_launch<T>(aa, m, rs, R, nseg, w, st);
            if (e != cudaSuccess) return e;
        }
        PROF_MARK(prof, KC_ATTENTION, 0, st);
        GemmArgs<T> go{};
        go.A = att; go.W = (const T*)L.w_o; go.bias = L.b_o; go.R = R; go.N = d; go.K = d;
        go.out_f = w.y; go.resid = w.x;
        PROF_MARK(prof, KC_GEMM_O, 1, st);
        k_gemm<T, EPI_RESID><<<grid(d), blk, 0, st>>>(go);
        PROF_MARK(prof, KC_GEMM_O, 0, st);
        PROF_MARK(prof, KC_LAYERNORM, 1, st);
        k_layernorm<T><<<(R + 7) / 8, 256, 0, st>>>(w.y, L.ln1_g, L.ln1_b, w.x, xb, R, d);
        PROF_MARK(prof, KC_LAYERNORM, 0, st);
        GemmArgs<T> g1{};
        g1.A = xb; g1.W = (const T*)L.w_1; g1.bias = L.b_1; g1.R = R; g1.N = F; g1.K = d;
        g1.out_t = hid;
        PROF_MARK(prof, KC_GEMM_FFN1, 1, st);
        k_gemm<T, EPI_RELU><<<grid(F), blk, 0, st>>>(g1);
        PROF_MARK(prof, KC_GEMM_FFN1, 0, st);
        GemmArgs<T> g2{};
        g2.A = hid; g2.W = (const T*)L.w_2; g2.bias = L.b_2; g2.R = R; g2.N = d; g2.K = F;
        g2.out_f = w.y; g2.resid = w.x;
        PROF_MARK(prof, KC_GEMM_FFN2, 1, st);
        k_gemm<T, EPI_RESID><<<grid(d), blk, 0, st>>>(g2);
        PROF_MARK(prof, KC_GEMM_FFN2, 0, st);
        PROF_MARK(prof, KC_LAYERNORM, 1, st);
        k_layernorm<T><<<(R + 7) / 8, 256, 0, st>>>(w.y, L.ln2_g, L.ln2_b, w.x, xb, R, d);
        PROF_MARK(prof, KC_LAYERNORM, 0, st);
        nl += 7;
    }
    if (want_heads && use_tc && tc->head) {
        PROF_MARK(prof, KC_HEAD, 1, st);
        const cudaError_t e = launch_head_tc(tc->head_hi, tc->head_lo, m, w, R, st);
        if (e != cudaSuccess) return e;
        PROF_MARK(prof, KC_HEAD, 0, st);
        nl += 1;
    } else if (want_heads) {
        PROF_MARK(prof, KC_HEAD, 1, st);
        if (use_tc && tc->head_g) {
            // e | V_k1 h + b_k1 on the tensor cores, fp32-accurate: h split
            // into bf16 parts (hi over xb, lo over att; both free after the
            // last layer), [E; V_k1] as stored in hi / lo parts
            k_split_rows<<<(unsigned)std::min<long long>(((long long)R * d / 2 + 255) / 256, 152 * 8), 256, 0, st>>>(
                w.x, (bf16*)w.xb, (bf16*)w.att, (long long)R * d / 2);
            TcGemmArgs g{};
            g.R = R; g.N = 4 * d; g.K = d; g.epi = EPI_TC_F32; g.bias = m.head_ek_b; g.out_f = w.hd4;
            g.split = 1; g.err = tc->err;
            const cudaError_t e =
                launch_gemm_tc_split(tc->a_xb, tc->a_att, tc->head_hi_g, tc->head_lo_g, g, tc->bn_head, st);
            if (e != cudaSuccess) return e;
            nl += 1;
        } else {
            // e | V_k1 h + b_k1 for all rows (fp32 tiled GEMM)
            GemmArgs<float> gh{};
            gh.A = w.x; gh.W = m.head_ek_w; gh.bias = m.head_ek_b; gh.R = R; gh.N = 4 * d; gh.K = d;
            gh.out_f = w.hd4;
            k_gemm<float, EPI_F32><<<dim3((4 * d + 63) / 64, (R + 63) / 64), 256, 0, st>>>(gh);
        }
        // then the small maps
        if (head_rows_supported(m) && !getenv("TPPSD_HEAD_OUT_WARP")) {
            const cudaError_t e = launch_head_rows(m, w, R, st);
            if (e != cudaSuccess) return e;
        } else {
            const int WO = m.head_width();
            const size_t wbytes = sizeof(float) * (size_t)d * WO;
            const int stage = wbytes <= 96 * 1024;
            const size_t sm = (stage ? wbytes : 0) + sizeof(float) * 8 * 4 * d;
            if (sm > 48 * 1024) cudaFuncSetAttribute(k_head_out, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
            const int blocks = min((R + 7) / 8, 152 * 2);
            k_head_out<<<blocks, 256, sm, st>>>(m, w, R, stage);
        }
        PROF_MARK(prof, KC_HEAD, 0, st);
        nl += 2;
    }
    if (launches) *launches += nl;
    return cudaGetLastError();
}

cudaError_t launch_forward(const DevModel& m, const KVCache& kv, const SeqState& ss, const Work& w,
                           const RowSpec& rs, bool want_heads, cudaStream_t st, int* launches,
                           const Prof* prof, const TcPlan* tc) {
    return m.dtype == 1 ? forward_t<bf16>(m, kv, ss, w, rs, want_heads, st, launches, prof, tc)
                        : forward_t<float>(m, kv, ss, w, rs, want_heads, st, launches, prof, tc);
}

cudaError_t launch_history_times(const SeqState& ss, int B, int H, cudaStream_t st) {
    k_history_times<<<(B + 127) / 128, 128, 0, st>>>(ss, B, H);
    return cudaGetLastError();
}

cudaError_t launch_begin(const CallParams& p, CallParams* dp, const SeqState& ss, DevStats* stats,
                         cudaStream_t st) {
    k_begin<<<(max(p.B, 1) + 255) / 256, 256, 0, st>>>(p, dp, ss, stats);
    return cudaGetLastError();
}

static size_t draft_buf_floats(const DevModel& m) {
    const int d = m.d, W = m.head_width();
    return (size_t)d * 11 + m.F + ((W + 3) & ~3) + 4 * (64 + 2) + 16;
}

size_t draft_smem_bytes(const DevModel& m, bool stage_weights) {
    const size_t wb = stage_weights ? ((m.bytes + 15) & ~(size_t)15) : 0;
    return wb + sizeof(float) * draft_buf_floats(m);
}

int draft_supported(const DevModel& m) {
    return (m.nh == 1 || m.nh == 2 || m.nh == 4) && (m.dh == 8 || m.dh == 16 || m.dh == 32 || m.dh == 64);
}

cudaError_t launch_draft(const DevModel& m, const KVCache& kv, const SeqState& ss,
                         const CallParams* dp, int B, int gamma, float* draft_heads, int gamma_max,
                         DevStats* stats, cudaStream_t st) {
    DraftArgs a{};
    a.m = m; a.kv = kv; a.ss = ss; a.P = dp; a.heads = draft_heads; a.st = stats;
    a.gamma = gamma; a.gamma_max = gamma_max;
    const size_t staged = draft_smem_bytes(m, true);
    a.stage = staged <= 200 * 1024;
    a.stage_bytes = a.stage ? (int)((m.bytes + 15) & ~(size_t)15) : 0;
    const size_t sm = draft_smem_bytes(m, a.stage);
    if (m.dtype == 1) {
        DISPATCH_DH(m.dh, {
            cudaFuncSetAttribute(k_draft<bf16, DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
            k_draft<bf16, DH><<<B, 128, sm, st>>>(a);
        });
    } else {
        DISPATCH_DH(m.dh, {
            cudaFuncSetAttribute(k_draft<float, DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
            k_draft<float, DH><<<B, 128, sm, st>>>(a);
        });
    }
    return cudaGetLastError();
}

cudaError_t launch_verify_epilogue(const DevModel& mT, const DevModel& mD, const SeqState& ss,
                                   const CallParams* dp, int B, int gamma, const float* t_heads,
                                   const float* d_heads, int gamma_max, DevStats* stats,
                                   cudaStream_t st, bool poisson) {
    EpiArgs a{};
    a.ss = ss; a.P = dp; a.th = t_heads; a.dh = d_heads;
    a.MT = mT.M; a.MD = mD.M; a.K = mT.K; a.WT = mT.head_width(); a.WD = mD.head_width();
    a.gamma = gamma; a.gamma_max = gamma_max; a.st = stats;
    a.poisson = poisson ? 1 : 0;
    return launch_k(k_verify_epilogue, dim3(B), dim3(128), 0, st, a);
}

cudaError_t launch_poisson_draft(const SeqState& ss, const CallParams* dp, int B, int gamma, int K,
                                 cudaStream_t st) {
    return launch_k(k_poisson_draft, dim3((B + 127) / 128), dim3(128), 0, st, ss, dp, gamma, K);
}

cudaError_t launch_ar_sample(const DevModel& mT, const SeqState& ss, const CallParams* dp, int B,
                             const float* heads, DevStats* stats, cudaStream_t st) {
    return launch_k(k_ar_sample, dim3((B + 127) / 128), dim3(128), 0, st, ss, dp, heads, mT.M, mT.K,
                    mT.head_width(), stats);
}

cudaError_t launch_round_control(const SeqState& ss, const CallParams* dp, int B, DevStats* stats,
                                 unsigned long long cond_handle, int use_cond, int* active_out,
                                 cudaStream_t st) {
    (void)B;
    return launch_k(k_round_control, dim3(1), dim3(256), 0, st, ss, dp, stats,
                    (cudaGraphConditionalHandle)cond_handle, use_cond, active_out);
}

cudaError_t launch_score_survival(const DevModel& m, const SeqState& ss, const Work& w, int B, int len,
                                  int g0, int rows, double t_end, double* out_logS, cudaStream_t st) {
    (void)B;
    if (rows <= 0) return cudaSuccess;
    k_score_survival<<<(rows + 127) / 128, 128, 0, st>>>(ss, w, m.M, m.K, len, g0, rows, t_end, out_logS);
    return cudaGetLastError();
}

cudaError_t launch_score_logs(const DevModel& m, const SeqState& ss, const Work& w, int B, int len,
                              int q, int g0, int rows, float* out_heads, float* out_logg, float* out_logf,
                              cudaStream_t st) {
    (void)B;
    if (rows <= 0) return cudaSuccess;
    k_score_logs<<<(rows + 127) / 128, 128, 0, st>>>(ss, w, m.M, m.K, len, q, g0, rows, out_heads,
                                                     out_logg, out_logf);
    return cudaGetLastError();
}

}  // namespace tppsd
