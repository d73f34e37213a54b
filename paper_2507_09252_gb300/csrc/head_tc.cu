// Target heads on the tensor cores (Sec. 4.2) for d = 128.  The four
// 128-column blocks of [E; V_k1] h feed disjoint head outputs: block 0 (e1)
// the component logits, 1 (e2) mu, 2 (e3) log sigma, 3 (V_k1 h + b_k1, then
// tanh) the mark logits.  So CTA (block nb, 128-row tile) computes block nb
// with tcgen05 and then its own head outputs, with no exchange between
// CTAs.  The head is fp32 arithmetic: h W^T is formed as
// h_hi W_hi + h_hi W_lo + h_lo W_hi with both operands split into two bf16
// parts (x = x_hi + x_lo), fp32 accumulation in TMEM (relative error about
// 2^-16 of |h| |W|).  Ten warps: warps 0-7 split the h rows (coalesced
// reads) into the two swizzled A operands and later own one row and 64 of
// its 128 accumulator columns each (warps w and w+4 share TMEM lanes
// 32 (w % 4)..); warp 8 loads the W_hi / W_lo tiles by TMA; one thread of
// warp 9 issues the MMAs.  The small output matrix is staged transposed
// ([output][128], rows padded to a multiple of 8 with zeros) so that a
// thread reads four weights per shared-memory load; the two column halves
// of a row meet through shared memory.
#include <cuda.h>

#include "common.cuh"
#include "engine.h"
#include "tc_ptx.cuh"

namespace tppsd {

struct HeadShape {
    static constexpr int D = 128, BM = 128, BK = 64, KB = D / BK;
    static constexpr int TILE = BM * BK * 2;  // 16 KB
    static constexpr int OFF_AH = 0, OFF_AL = KB * TILE, OFF_BH = 2 * KB * TILE, OFF_BL = 3 * KB * TILE;
    static constexpr int OFF_BAR = 4 * KB * TILE;
    static constexpr int OFF_PART = OFF_BAR + 64;               // [BM][8] partial sums of column half 1
    static constexpr int OFF_W = OFF_PART + BM * 8 * 4;         // [cntp][D] outputs, bias [cntp], b_k1 [D]
    __host__ __device__ static constexpr int cntp(int cnt) { return (cnt + 7) & ~7; }
    __host__ __device__ static constexpr size_t smem_bytes(int cnt) {
        return (size_t)OFF_W + ((size_t)cntp(cnt) * D + cntp(cnt) + D) * 4 + 1024;
    }
};

__device__ __forceinline__ void head_epi_sync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

__global__ void __launch_bounds__(320, 1)
    k_head_tc(const __grid_constant__ CUtensorMap mapHi, const __grid_constant__ CUtensorMap mapLo, DevModel m,
              Work w, int R) {
    using S = HeadShape;
    constexpr int D = S::D;
    // the weight tiles (never written by a sampling kernel) are requested
    // before griddepcontrol.wait; the rows and outputs only after it
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* bars = (uint64_t*)(smem + S::OFF_BAR);
    uint64_t* a_ready = bars;      // both A operands written (256 arrivals)
    uint64_t* b_full = bars + 1;   // W tiles landed
    uint64_t* done = bars + 2;     // accumulator complete
    uint32_t* tslot = (uint32_t*)(bars + 3);
    float* part = (float*)(smem + S::OFF_PART);
    float* ws = (float*)(smem + S::OFF_W);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nb = blockIdx.x, m0 = blockIdx.y * S::BM, rows = min(S::BM, R - m0);
    if (threadIdx.x == 0) {
        mbar_init(a_ready, 256);
        mbar_init(b_full, 1);
        mbar_init(done, 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(tslot, 128);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;

    if (warp == 8) {
        if (lane == 0) {
            mbar_arrive_expect_tx(b_full, 2 * S::KB * S::TILE);
            for (int kb = 0; kb < S::KB; ++kb) {
                tma_load_2d(smem + S::OFF_BH + kb * S::TILE, &mapHi, b_full, kb * S::BK, nb * 128);
                tma_load_2d(smem + S::OFF_BL + kb * S::TILE, &mapLo, b_full, kb * S::BK, nb * 128);
            }
        }
    } else if (warp == 9) {
        if (lane == 0) {
            bool ok = mbar_wait(a_ready, 0, w.err, 51);
            ok = ok && mbar_wait(b_full, 0, w.err, 52);
            tc_fence_after();
            if (ok) {
                const uint32_t idesc = idesc_bf16(128, 128);
                const uint32_t ah = smem_u32(smem + S::OFF_AH), al = smem_u32(smem + S::OFF_AL);
                const uint32_t bh = smem_u32(smem + S::OFF_BH), bl = smem_u32(smem + S::OFF_BL);
                for (int kb = 0; kb < S::KB; ++kb)
#pragma unroll
                    for (int kk = 0; kk < S::BK / 16; ++kk) {
                        const uint32_t o = kb * S::TILE + kk * 32;
                        tc_mma_bf16(tmem, sw128_desc(ah + o), sw128_desc(bh + o), idesc, (kb | kk) != 0);
                        tc_mma_bf16(tmem, sw128_desc(ah + o), sw128_desc(bl + o), idesc, 1u);
                        tc_mma_bf16(tmem, sw128_desc(al + o), sw128_desc(bh + o), idesc, 1u);
                    }
            }
            tc_commit(done);
        }
    } else {
        const int tid = threadIdx.x;
        pdl_wait();
        // A operands: h rows split into hi / lo bf16, written in the swizzled
        // K-major layout (16-byte chunk c of row r at chunk c ^ (r & 7)); all
        // 16 global loads of a thread are issued before the first store
        constexpr int NV = S::BM * D / 4 / 256;
        {
            float4 xv[NV];
#pragma unroll
            for (int j = 0; j < NV; ++j) {
                const int f = tid + j * 256, r = f >> 5, c4 = f & 31;
                xv[j] = r < rows ? *reinterpret_cast<const float4*>(w.x + (size_t)(m0 + r) * D + 4 * c4)
                                 : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int j = 0; j < NV; ++j) {
                const int f = tid + j * 256, r = f >> 5, c4 = f & 31;
                const float xs[4] = {xv[j].x, xv[j].y, xv[j].z, xv[j].w};
                uint32_t hi[2], lo[2];
#pragma unroll
                for (int i = 0; i < 2; ++i) {
                    const __nv_bfloat162 h2 = __floats2bfloat162_rn(xs[2 * i], xs[2 * i + 1]);
                    const float2 hf = __bfloat1622float2(h2);
                    const __nv_bfloat162 l2 = __floats2bfloat162_rn(xs[2 * i] - hf.x, xs[2 * i + 1] - hf.y);
                    hi[i] = *reinterpret_cast<const uint32_t*>(&h2);
                    lo[i] = *reinterpret_cast<const uint32_t*>(&l2);
                }
                const int kb = c4 >> 4, ch = (c4 & 15) >> 1, half = c4 & 1;
                const int off = kb * S::TILE + r * 128 + ((ch ^ (r & 7)) << 4) + half * 8;
                *reinterpret_cast<uint2*>(smem + S::OFF_AH + off) = make_uint2(hi[0], hi[1]);
                *reinterpret_cast<uint2*>(smem + S::OFF_AL + off) = make_uint2(lo[0], lo[1]);
            }
        }
        fence_proxy_async_smem();
        mbar_arrive(a_ready);
        // while the tensor cores run: this block's output matrix (columns
        // col0.. of the [d][3M+K] head map) transposed into [cntp][D], its
        // bias and b_k1
        const int M = m.M, K = m.K, WO = 3 * M + K;
        const int cnt = nb < 3 ? M : K, col0 = nb < 3 ? nb * M : 3 * M, cp = S::cntp(cnt);
        float* wb = ws + cp * D;
        float* bk1 = wb + cp;
        for (int i0 = tid; i0 < cp * D; i0 += 8 * 256) {  // batches of 8 loads per thread
            float v[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int i = i0 + j * 256, o = i / D, c = i % D;
                v[j] = i < cp * D && o < cnt ? m.head_out_t[(size_t)c * WO + col0 + o] : 0.f;
            }
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (i0 + j * 256 < cp * D) ws[i0 + j * 256] = v[j];
        }
        for (int i = tid; i < cp; i += 256) wb[i] = i < cnt ? m.head_out_b[col0 + i] : 0.f;
        for (int i = tid; i < D; i += 256) bk1[i] = m.head_ek_b[3 * D + i];
        head_epi_sync();
        // row t of the tile, accumulator columns 64 hf .. 64 hf + 63
        const int q = warp & 3, hf = warp >> 2, t = q * 32 + lane;
        const bool live = t < rows && w.row_seq[m0 + t] >= 0;
        mbar_wait(done, 0, w.err, 53);
        tc_fence_after();
        pdl_trigger();  // the next kernel may be scheduled while the outputs are formed
        float v[64];
        tmem_ld64(tmem + ((uint32_t)(q * 32) << 16) + 64 * hf, v);
        if (nb == 3) {
#pragma unroll
            for (int i = 0; i < 64; ++i) v[i] = tanhf(v[i] + bk1[64 * hf + i]);
        }
        float* dst = w.heads + (size_t)(m0 + t) * WO + col0;
        const bool norm = nb == 0 || nb == 3;  // log w, log f: subtract log sum exp
        float mx = -INFINITY, sum = 0.f;
        for (int o0 = 0; o0 < cp; o0 += 8) {
            float acc[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const float4* wr = reinterpret_cast<const float4*>(ws + (o0 + j) * D + 64 * hf);
                float a0 = 0.f, a1 = 0.f;
#pragma unroll
                for (int i = 0; i < 16; i += 2) {
                    const float4 w0 = wr[i], w1 = wr[i + 1];
                    a0 = fmaf(w0.x, v[4 * i], a0);
                    a0 = fmaf(w0.y, v[4 * i + 1], a0);
                    a0 = fmaf(w0.z, v[4 * i + 2], a0);
                    a0 = fmaf(w0.w, v[4 * i + 3], a0);
                    a1 = fmaf(w1.x, v[4 * i + 4], a1);
                    a1 = fmaf(w1.y, v[4 * i + 5], a1);
                    a1 = fmaf(w1.z, v[4 * i + 6], a1);
                    a1 = fmaf(w1.w, v[4 * i + 7], a1);
                }
                acc[j] = a0 + a1;
            }
            if (hf == 1) {
#pragma unroll
                for (int j = 0; j < 8; ++j) part[t * 8 + j] = acc[j];
            }
            head_epi_sync();
            if (hf == 0) {
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[j] = wb[o0 + j] + (acc[j] + part[t * 8 + j]);
                if (norm) {
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        if (o0 + j >= cnt) continue;
                        const float mn = fmaxf(mx, acc[j]);
                        sum = sum * expf(mx - mn) + expf(acc[j] - mn);
                        mx = mn;
                    }
                }
                if (live) {
                    const float sub = norm && cp == 8 ? mx + logf(sum) : 0.f;  // one chunk: final here
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        if (o0 + j < cnt) dst[o0 + j] = acc[j] - sub;
                }
            }
            head_epi_sync();  // part is rewritten by the next chunk
        }
        if (hf == 0 && live && norm && cp > 8) {  // several chunks: normalise what was written
            const float lz = mx + logf(sum);
            for (int o = 0; o < cnt; ++o) dst[o] -= lz;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 128);
    pdl_trigger();
}

int head_tc_supported(const DevModel& m) {
    const int cnt = m.M > m.K ? m.M : m.K;
    return m.dtype == 1 && m.d == HeadShape::D && HeadShape::smem_bytes(cnt) <= 227 * 1024;
}

cudaError_t launch_head_tc(const CUtensorMap& hi, const CUtensorMap& lo, const DevModel& m, const Work& w, int R,
                           cudaStream_t st) {
    if (R <= 0) return cudaSuccess;
    if (!head_tc_supported(m)) return cudaErrorInvalidValue;
    const size_t sm = HeadShape::smem_bytes(m.M > m.K ? m.M : m.K);
    cudaError_t e = cudaFuncSetAttribute(k_head_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    return launch_k(k_head_tc, dim3(4, (R + 127) / 128), dim3(320), sm, st, hi, lo, m, w, R);
}

}  // namespace tppsd
