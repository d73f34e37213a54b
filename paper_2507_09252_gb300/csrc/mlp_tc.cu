// Fused post-attention block of one target layer on the tensor cores (bf16
// operands, fp32 accumulation in TMEM), for d = 128 (reading of the layer:
// post-LN Transformer block, ReLU FFN):
//   x1 = LN1(x + att W_o^T + b_o)
//   x  = LN2(x1 + relu(x1 W_1^T + b_1) W_2^T + b_2),   xb = bf16(x)
// One CTA per 128-row tile, ten warps:
//   warp 8     producer: the attention tile and every weight tile (TMA,
//              128-byte swizzle) through a ring of stages
//   warp 9     one thread issues tcgen05.mma; W tiles are consumed in the
//              order O-proj, H_0, H_1, F2_0, H_2, F2_1, ... so the tensor
//              core computes the next FFN1 chunk while the epilogue warps
//              turn the current one into bf16 ReLU activations
//   warps 0-7  epilogues: warps w and w+4 share TMEM lanes 32(w%4).. (row t
//              = lane), each taking 64 of the row's 128 columns; LayerNorm
//              partial sums meet in shared memory.  The residual tile is
//              read and the output tile written with coalesced accesses
//              through shared memory.
// TMEM (512 columns): 0-127 the output projection, then (once LN1 has read
// it) the FFN2 accumulator; 128-383 two FFN1 chunk buffers; 384-511 x1 in
// fp32 (the LN2 residual).  Shared memory: the attention tile, then x1 in
// bf16 (A operand of FFN1); the residual tile, then two buffers of chunk
// activations (A operand of FFN2), then the output tile; the weight ring.
// The FFN hidden layer (F columns) never leaves the SM.  Every wait is
// bounded.
#include <cuda.h>

#include "common.cuh"
#include "engine.h"
#include "tc_ptx.cuh"

namespace tppsd {

struct MlpShape {
    static constexpr int D = 128, BM = 128, BK = 64, CH = 128;
    static constexpr int TILE = BM * BK * 2;            // 128 rows x 64 bf16 (16 KB)
    static constexpr int STAGES = 6;
    static constexpr int RLD = D + 4;                   // padded fp32 row (floats)
    static constexpr int PF = 1024;                     // largest FFN width
    static constexpr int OFF_A = 0;                     // attention tile, then x1 (2 k-blocks)
    static constexpr int OFF_R = OFF_A + 2 * TILE;      // residual / 2 activation buffers / output
    static constexpr int R_BYTES = ((BM * RLD * 4 + 1023) / 1024) * 1024;
    static constexpr int OFF_W = OFF_R + R_BYTES;       // weight ring
    static constexpr int OFF_P = OFF_W + STAGES * TILE; // b_o g1 be1 b_2 g2 be2 (D each), b_1 (F)
    static constexpr int OFF_RED = OFF_P + (6 * D + PF) * 4;  // LayerNorm partials [2][4][BM]
    static constexpr int OFF_B = OFF_RED + 8 * BM * 4;
    static constexpr int NBAR = 23;
    static constexpr size_t SMEM = (size_t)OFF_B + NBAR * 8 + 16 + 1024;
    static_assert(R_BYTES >= 4 * TILE, "two activation buffers fit in the residual region");
};

// 16 consecutive columns c0.. of row t as bf16 into a K-major operand tile
// pair (two 64-column k-blocks), 128-byte swizzle: the 16-byte chunk c of
// row t sits at chunk c ^ (t & 7) of the row's 128 bytes.
__device__ __forceinline__ void st_swizzled16(unsigned char* tiles, int t, int c0, const float* v) {
    uint32_t w[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const __nv_bfloat162 p = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
        w[i] = *reinterpret_cast<const uint32_t*>(&p);
    }
    const int kb = c0 >> 6, ch = (c0 & 63) >> 3;
    unsigned char* row = tiles + kb * MlpShape::TILE + t * 128;
    *reinterpret_cast<uint4*>(row + (((ch + 0) ^ (t & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
    *reinterpret_cast<uint4*>(row + (((ch + 1) ^ (t & 7)) << 4)) = make_uint4(w[4], w[5], w[6], w[7]);
}

__device__ __forceinline__ void epi_sync() {  // the 256 epilogue threads only
    asm volatile("bar.sync 1, 256;" ::: "memory");
}
__device__ __forceinline__ void epi_sync512() {  // the cluster form's 512 epilogue threads
    asm volatile("bar.sync 1, 512;" ::: "memory");
}

__global__ void __launch_bounds__(320, 1)
    k_mlp_tc(const __grid_constant__ CUtensorMap mapAtt, const __grid_constant__ CUtensorMap mapWo,
             const __grid_constant__ CUtensorMap mapW1, const __grid_constant__ CUtensorMap mapW2, MlpArgs a) {
    using S = MlpShape;
    constexpr int D = S::D;
    pdl_wait();
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* A = smem + S::OFF_A;
    unsigned char* Rg = smem + S::OFF_R;
    float* res = (float*)Rg;
    unsigned char* Wr = smem + S::OFF_W;
    float* prm = (float*)(smem + S::OFF_P);
    float* red = (float*)(smem + S::OFF_RED);
    uint64_t* bars = (uint64_t*)(smem + S::OFF_B);
    uint64_t* full = bars;            // [STAGES]
    uint64_t* empty = bars + 6;       // [STAGES]
    uint64_t* abar = bars + 12;       // attention tile landed
    uint64_t* o_done = bars + 13;     // output projection in TMEM
    uint64_t* x1_ready = bars + 14;   // x1 operand written (256 arrivals)
    uint64_t* h_done = bars + 15;     // [2] FFN1 chunk j in TMEM buffer j & 1
    uint64_t* e2_done = bars + 17;    // [2] chunk j's activations in buffer j & 1 (256 arrivals)
    uint64_t* hid_free = bars + 19;   // [2] FFN2 of chunk j done: buffer j & 1 reusable
    uint64_t* y_done = bars + 21;     // FFN2 accumulator complete
    uint32_t* tslot = (uint32_t*)(bars + 22);
    static_assert(S::STAGES <= 6, "barrier slots");
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * S::BM, rows = min(S::BM, a.R - m0);
    const int nc = a.F / S::CH;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(abar, 1);
        mbar_init(o_done, 1);
        mbar_init(x1_ready, 256);
        for (int b = 0; b < 2; ++b) {
            mbar_init(&h_done[b], 1);
            mbar_init(&e2_done[b], 256);
            mbar_init(&hid_free[b], 1);
        }
        mbar_init(y_done, 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(tslot, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;

    if (warp == 8) {
        if (lane == 0) {
            mbar_arrive_expect_tx(abar, 2 * S::TILE);
            tma_load_2d(A, &mapAtt, abar, 0, m0);
            tma_load_2d(A + S::TILE, &mapAtt, abar, 64, m0);
            int q = 0;
            bool ok = true;
            auto load_w = [&](const CUtensorMap* map, int x, int y) {
                if (!ok) return;
                const int s = q % S::STAGES, round = q / S::STAGES;
                ok = mbar_wait(&empty[s], (round & 1) ^ 1, a.err, 31);
                if (!ok) return;
                mbar_arrive_expect_tx(&full[s], S::TILE);
                tma_load_2d(Wr + s * S::TILE, map, &full[s], x, y);
                ++q;
            };
            load_w(&mapWo, 0, 0);
            load_w(&mapWo, 64, 0);
            load_w(&mapW1, 0, 0);
            load_w(&mapW1, 64, 0);
            for (int j = 0; j < nc; ++j) {
                if (j + 1 < nc) {
                    load_w(&mapW1, 0, (j + 1) * S::CH);
                    load_w(&mapW1, 64, (j + 1) * S::CH);
                }
                load_w(&mapW2, j * S::CH, 0);
                load_w(&mapW2, j * S::CH + 64, 0);
            }
        }
    } else if (warp == 9) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(128, 128);
            int q = 0;
            bool ok = true;
            // one 128x128x64 step: A k-block at a_addr, W tile from the ring
            auto mma_tile = [&](uint32_t a_addr, uint32_t d_tmem, bool acc) {
                if (!ok) return;
                const int s = q % S::STAGES, round = q / S::STAGES;
                ok = mbar_wait(&full[s], round & 1, a.err, 32);
                if (!ok) return;
                tc_fence_after();
                const uint32_t b_addr = smem_u32(Wr + s * S::TILE);
#pragma unroll
                for (int kk = 0; kk < S::BK / 16; ++kk)
                    tc_mma_bf16(d_tmem, sw128_desc(a_addr + kk * 32), sw128_desc(b_addr + kk * 32), idesc,
                                (acc || kk) ? 1u : 0u);
                tc_commit(&empty[s]);
                ++q;
            };
            const uint32_t a0 = smem_u32(A), r0 = smem_u32(Rg);
            ok = mbar_wait(abar, 0, a.err, 33);
            tc_fence_after();
            mma_tile(a0, tmem, false);
            mma_tile(a0 + S::TILE, tmem, true);
            tc_commit(o_done);
            if (ok) ok = mbar_wait(x1_ready, 0, a.err, 34);
            tc_fence_after();
            auto ffn1 = [&](int j) {
                const uint32_t hb = tmem + 128 + (uint32_t)(j & 1) * 128;
                mma_tile(a0, hb, false);
                mma_tile(a0 + S::TILE, hb, true);
                tc_commit(&h_done[j & 1]);
            };
            ffn1(0);
            for (int j = 0; j < nc; ++j) {
                if (j + 1 < nc) ffn1(j + 1);  // its TMEM buffer was released by chunk j-1's epilogue
                if (ok) ok = mbar_wait(&e2_done[j & 1], (j >> 1) & 1, a.err, 35);
                tc_fence_after();
                const uint32_t hs = r0 + (uint32_t)(j & 1) * 2 * S::TILE;
                mma_tile(hs, tmem, j > 0);
                mma_tile(hs + S::TILE, tmem, true);
                tc_commit(&hid_free[j & 1]);
            }
            tc_commit(y_done);
        }
    } else {
        // epilogue warps 0-7: row t = 32 (warp % 4) + lane, columns cb..cb+63
        const int tid = threadIdx.x, q = warp & 3, hh = warp >> 2, t = q * 32 + lane, cb = hh * 64;
        const bool live = t < rows;
        // residual tile (coalesced: float4 f of the tile is row f / 32) and the
        // epilogue parameters; all loads are issued before any store
        {
            constexpr int NV = S::BM * D / 4 / 256;  // 16 float4 per thread
            float4 v[NV];
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int f = tid + 256 * k, r = f >> 5, c4 = f & 31;
                v[k] = r < rows ? *reinterpret_cast<const float4*>(a.x + (size_t)(m0 + r) * D + 4 * c4)
                                : make_float4(0.f, 0.f, 0.f, 0.f);
            }
            const float* src[6] = {a.b_o, a.ln1_g, a.ln1_b, a.b_2, a.ln2_g, a.ln2_b};
            float pv[3];
#pragma unroll
            for (int k = 0; k < 3; ++k) {
                const int i = tid + 256 * k;  // 768 = 6 D vector entries
                pv[k] = src[i / D][i % D];
            }
            float b1v[S::PF / 256];
#pragma unroll
            for (int k = 0; k < S::PF / 256; ++k) {
                const int i = tid + 256 * k;
                b1v[k] = i < a.F ? a.b_1[i] : 0.f;
            }
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int f = tid + 256 * k, r = f >> 5, c4 = f & 31;
                *reinterpret_cast<float4*>(res + r * S::RLD + 4 * c4) = v[k];
            }
#pragma unroll
            for (int k = 0; k < 3; ++k) prm[tid + 256 * k] = pv[k];
#pragma unroll
            for (int k = 0; k < S::PF / 256; ++k) prm[6 * D + tid + 256 * k] = b1v[k];
        }
        epi_sync();
        const float *p_bo = prm + cb, *p_g1 = prm + D + cb, *p_be1 = prm + 2 * D + cb, *p_b2 = prm + 3 * D + cb;
        const float *p_g2 = prm + 4 * D + cb, *p_be2 = prm + 5 * D + cb, *p_b1 = prm + 6 * D + cb;
        const uint32_t tl = tmem + ((uint32_t)(q * 32) << 16);
        float* xr = res + t * S::RLD + cb;
        // mean and 1/sqrt(var + eps) of a row whose halves are held by the
        // thread pairs (t, hh = 0 / 1); rd: this LayerNorm's [4][BM] partials
        auto row_stats = [&](const float* y, float* rd, float& mean, float& inv) {
            float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
            for (int c = 0; c < 64; c += 4) {
                s0 += y[c];
                s1 += y[c + 1];
                s2 += y[c + 2];
                s3 += y[c + 3];
            }
            rd[hh * S::BM + t] = (s0 + s1) + (s2 + s3);
            epi_sync();
            mean = (rd[t] + rd[S::BM + t]) / D;
            s0 = s1 = s2 = s3 = 0.f;
#pragma unroll
            for (int c = 0; c < 64; c += 4) {
                s0 = fmaf(y[c] - mean, y[c] - mean, s0);
                s1 = fmaf(y[c + 1] - mean, y[c + 1] - mean, s1);
                s2 = fmaf(y[c + 2] - mean, y[c + 2] - mean, s2);
                s3 = fmaf(y[c + 3] - mean, y[c + 3] - mean, s3);
            }
            rd[(2 + hh) * S::BM + t] = (s0 + s1) + (s2 + s3);
            epi_sync();
            inv = 1.0f / sqrtf((rd[2 * S::BM + t] + rd[3 * S::BM + t]) / D + LN_EPS);
        };
        mbar_wait(o_done, 0, a.err, 37);
        tc_fence_after();
        // y = O + b_o + x; LN1 -> x1: fp32 into TMEM columns 384.., bf16 into
        // the A operand of FFN1 (columns cb.. are k-block hh)
        float y[64];
        tmem_ld64(tl + cb, y);
#pragma unroll
        for (int c = 0; c < 64; c += 4) {
            const float4 r4 = *reinterpret_cast<const float4*>(xr + c);
            y[c] += p_bo[c] + r4.x;
            y[c + 1] += p_bo[c + 1] + r4.y;
            y[c + 2] += p_bo[c + 2] + r4.z;
            y[c + 3] += p_bo[c + 3] + r4.w;
        }
        float mean, inv;
        row_stats(y, red, mean, inv);  // its barriers also end every read of the residual tile
#pragma unroll
        for (int c = 0; c < 64; ++c) y[c] = live ? (y[c] - mean) * inv * p_g1[c] + p_be1[c] : 0.f;
        tmem_st64(tl + 384 + cb, y);
#pragma unroll
        for (int c0 = 0; c0 < 64; c0 += 16) st_swizzled16(A, t, cb + c0, y + c0);
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(x1_ready);
        // FFN1 chunks: ReLU(H + b_1) -> bf16 operand of FFN2, buffer j & 1
        for (int j = 0; j < nc; ++j) {
            mbar_wait(&h_done[j & 1], (j >> 1) & 1, a.err, 38);
            if (j >= 2) mbar_wait(&hid_free[j & 1], ((j >> 1) - 1) & 1, a.err, 39);
            tc_fence_after();
            tmem_ld64(tl + 128 + (uint32_t)(j & 1) * 128 + cb, y);
            const float* b1 = p_b1 + j * S::CH;
#pragma unroll
            for (int c = 0; c < 64; ++c) y[c] = fmaxf(y[c] + b1[c], 0.f);
            unsigned char* hs = Rg + (j & 1) * 2 * S::TILE;
#pragma unroll
            for (int c0 = 0; c0 < 64; c0 += 16) st_swizzled16(hs, t, cb + c0, y + c0);
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(&e2_done[j & 1]);
        }
        // LN2 over y = F2 + b_2 + x1
        mbar_wait(y_done, 0, a.err, 40);
        tc_fence_after();
        float x1[64];
        tmem_ld64(tl + cb, y);
        tmem_ld64(tl + 384 + cb, x1);
#pragma unroll
        for (int c = 0; c < 64; ++c) y[c] += p_b2[c] + x1[c];
        row_stats(y, red + 4 * S::BM, mean, inv);
        // output tile through shared memory (the activation buffers are free:
        // every FFN2 step has completed), then coalesced row writes
#pragma unroll
        for (int c = 0; c < 64; c += 4) {
            float4 o;
            o.x = (y[c] - mean) * inv * p_g2[c] + p_be2[c];
            o.y = (y[c + 1] - mean) * inv * p_g2[c + 1] + p_be2[c + 1];
            o.z = (y[c + 2] - mean) * inv * p_g2[c + 2] + p_be2[c + 2];
            o.w = (y[c + 3] - mean) * inv * p_g2[c + 3] + p_be2[c + 3];
            *reinterpret_cast<float4*>(xr + c) = o;
        }
        epi_sync();
        {
            constexpr int NV = S::BM * D / 4 / 256;
            float4 v[NV];
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int f = tid + 256 * k, r = f >> 5, c4 = f & 31;
                v[k] = *reinterpret_cast<const float4*>(res + r * S::RLD + 4 * c4);
            }
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int f = tid + 256 * k, r = f >> 5, c4 = f & 31;
                if (r >= rows) continue;
                *reinterpret_cast<float4*>(a.x + (size_t)(m0 + r) * D + 4 * c4) = v[k];
                const __nv_bfloat162 p0 = __floats2bfloat162_rn(v[k].x, v[k].y);
                const __nv_bfloat162 p1 = __floats2bfloat162_rn(v[k].z, v[k].w);
                uint2 w;
                w.x = *reinterpret_cast<const uint32_t*>(&p0);
                w.y = *reinterpret_cast<const uint32_t*>(&p1);
                *reinterpret_cast<uint2*>(a.xb + (size_t)(m0 + r) * D + 4 * c4) = w;
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 512);
    pdl_trigger();
}

// ---------------------------------------------------------------------------
// Cluster form of the same block: the F hidden columns are split over a
// cluster of F / 128 CTAs (at most 8) that share one 128-row tile.  CTA c
// of the cluster computes the output projection and LN1 of the tile (every
// CTA the same values, the same instructions on the same inputs), FFN1
// chunk c with its ReLU, and the partial FFN2 product of that chunk; CTA 0
// adds x1 + b_2 to its partial.  The partials meet through distributed
// shared memory: each CTA pushes row slice p of its partial to CTA p with
// one bulk copy (into the weight region, free once every CTA's FFN2 is
// done); CTA c sums rows 128c/n .. of all n partials (in CTA order),
// applies LN2 and writes them.  The dependent chain of one CTA is
// thus one FFN1 chunk and one FFN2 chunk instead of F / 128 of each, and
// the weights a CTA streams drop to W_o plus 1/n of W_1 and W_2 (six tiles,
// all in flight at once).  Eighteen warps: sixteen epilogue warps (warp w
// reads TMEM lanes 32 (w % 4).. and takes 32 of its rows' 128 columns, so
// each element-wise phase is a quarter row per thread), a producer warp
// (TMA) and an MMA warp.  TMEM: 0-127 the output projection, then the
// FFN2 partial; 128-255 the FFN1 chunk; 256-383 x1 in fp32; 384.. the next
// layer's Q, K, V slice.
//
// With a.qkv the block also computes the next layer's Q, K and V (the QKV
// GEMM of the next layer folded in): CTA c writes its finished rows (bf16)
// into the A tile at their row offset, sends that slice (one contiguous
// 128-byte-per-row block per k-block under the 128-byte swizzle) to every
// peer by bulk copy, and once the whole 128-row tile is in place multiplies
// it by columns c NQ .. (c+1) NQ - 1 of W_qkv (NQ = 3d / n, prefetched at
// start); the epilogue adds the bias, rounds to bf16 and scatters Q to the
// row buffer and K, V into the cache, as the QKV GEMM does.
struct MlpClShape {
    static constexpr int D = 128, BM = 128, BK = 64, CH = 128;
    static constexpr int TILE = BM * BK * 2;
    static constexpr int NT = 6;                           // W_o, W_1 chunk, W_2 chunk: 2 tiles each
    static constexpr int RLD = D + 4;
    static constexpr int OFF_A = 0;                        // attention tile, then x1 (bf16)
    static constexpr int OFF_R = OFF_A + 2 * TILE;         // residual, then activations, then partial
    static constexpr int R_BYTES = ((BM * RLD * 4 + 1023) / 1024) * 1024;
    static constexpr int OFF_W = OFF_R + R_BYTES;
    static constexpr int OFF_P = OFF_W + NT * TILE;        // b_o g1 be1 b_2 g2 be2 (D each), b_1 chunk
    static constexpr int OFF_RED = OFF_P + (6 * D + CH) * 4;
    static constexpr int OFF_B = OFF_RED + 8 * BM * 4;     // LN1 partials: [sum, centred squares][4][BM]
    // sixteen epilogue warps (lane quarter q = warp % 4, column quarter
    // warp / 4: 32 columns per thread), then the producer and MMA warps
    static constexpr int EW = 16, ET = 32 * EW, CW = D / (EW / 4), THREADS = 32 * (EW + 2);
    static constexpr int NBAR = 18;
    __host__ __device__ static constexpr int SLICE_BYTES(int ncl) { return (BM / ncl) * RLD * 4; }
    static_assert(NT * TILE >= BM * RLD * 4, "the partial slices fit in the weight region");
    // next layer's W_qkv columns of this CTA: 3D / ncl rows of 128 B per k-block
    static constexpr int OFF_Q = ((OFF_B + NBAR * 8 + 16 + 1023) / 1024) * 1024;
    __host__ __device__ static constexpr int NQ(int ncl) { return 3 * D / ncl; }
    __host__ __device__ static constexpr bool QKV_OK(int ncl) { return ncl == 4 || ncl == 8; }
    static constexpr size_t SMEM = (size_t)OFF_Q + 2 * 96 * 128 + 1024;  // room for NQ <= 96
    static_assert(R_BYTES >= 2 * TILE, "the activation tile fits in the residual region");
    static_assert(SMEM <= 227 * 1024, "shared memory");
    static_assert(SMEM <= 227 * 1024, "shared memory");
};

// 8 consecutive columns c0.. (c0 % 8 == 0) of row t of a pair of
// 128-byte-swizzled 64-column tiles, rounded to bf16.
__device__ __forceinline__ void st_swizzled8(unsigned char* tiles, int t, int c0, const float* v) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const __nv_bfloat162 p = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
        w[i] = *reinterpret_cast<const uint32_t*>(&p);
    }
    const int kb = c0 >> 6, ch = (c0 & 63) >> 3;
    unsigned char* row = tiles + kb * MlpShape::TILE + t * 128;
    *reinterpret_cast<uint4*>(row + ((ch ^ (t & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
}

// 4 consecutive columns c0.. (c0 % 4 == 0) of row t, the same layout.
__device__ __forceinline__ void st_swizzled4(unsigned char* tiles, int t, int c0, const float* v) {
    const __nv_bfloat162 p0 = __floats2bfloat162_rn(v[0], v[1]);
    const __nv_bfloat162 p1 = __floats2bfloat162_rn(v[2], v[3]);
    const int kb = c0 >> 6, ch = (c0 & 63) >> 3;
    unsigned char* row = tiles + kb * MlpShape::TILE + t * 128;
    *reinterpret_cast<uint2*>(row + ((ch ^ (t & 7)) << 4) + (c0 & 4) * 2) =
        make_uint2(*reinterpret_cast<const uint32_t*>(&p0), *reinterpret_cast<const uint32_t*>(&p1));
}

template <int NCL>
__global__ void __launch_bounds__(MlpClShape::THREADS, 1)
    k_mlp_cl(const __grid_constant__ CUtensorMap mapAtt, const __grid_constant__ CUtensorMap mapWo,
             const __grid_constant__ CUtensorMap mapW1, const __grid_constant__ CUtensorMap mapW2,
             const __grid_constant__ CUtensorMap mapWq, MlpArgs a) {
    using S = MlpClShape;
    constexpr int D = S::D;
    // griddepcontrol.wait comes after everything that reads no output of the
    // previous kernel: barrier set-up, TMEM allocation, the weight tiles and
    // the bias / LayerNorm parameters (never written by a sampling kernel)
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* A = smem + S::OFF_A;
    unsigned char* Rg = smem + S::OFF_R;
    float* res = (float*)Rg;     // residual tile, later this CTA's FFN2 partial [BM][RLD]
    unsigned char* Wt = smem + S::OFF_W;
    float* prm = (float*)(smem + S::OFF_P);
    float* red = (float*)(smem + S::OFF_RED);
    uint64_t* bars = (uint64_t*)(smem + S::OFF_B);
    uint64_t* full = bars;            // [NT] weight tile i landed
    uint64_t* abar = bars + 6;        // attention tile landed
    uint64_t* o_done = bars + 7;      // output projection in TMEM
    uint64_t* x1_ready = bars + 8;    // x1 operand written (ET arrivals)
    uint64_t* h_done = bars + 9;      // FFN1 chunk in TMEM
    uint64_t* e2_done = bars + 10;    // chunk activations written (ET arrivals)
    uint64_t* y_done = bars + 11;     // FFN2 partial in TMEM
    uint64_t* rbar = bars + 12;       // the other CTAs' partial slices landed
    uint64_t* wqbar = bars + 13;      // next layer's W_qkv columns landed
    uint64_t* qa_local = bars + 14;   // this CTA's rows written into the A tile (ET arrivals)
    uint64_t* qa_remote = bars + 15;  // the other CTAs' rows landed in the A tile
    uint64_t* q_done = bars + 16;     // next layer's Q, K, V slice in TMEM
    uint32_t* tslot = (uint32_t*)(bars + 17);
    unsigned char* Wq = smem + S::OFF_Q;
    constexpr int NQ = S::NQ(NCL), RW = S::BM / NCL;
    constexpr int ET = S::ET, CW = S::CW, WP = S::EW, WM = S::EW + 1;  // producer, MMA warps
    const bool qkv = S::QKV_OK(NCL) && a.qkv;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = (int)cluster_ctarank();
    const int m0 = blockIdx.y * S::BM, rows = min(S::BM, a.R - m0);

    if (threadIdx.x == 0) {
        for (int i = 0; i < S::NT; ++i) mbar_init(&full[i], 1);
        mbar_init(abar, 1);
        mbar_init(o_done, 1);
        mbar_init(x1_ready, ET);
        mbar_init(h_done, 1);
        mbar_init(e2_done, ET);
        mbar_init(y_done, 1);
        mbar_init(rbar, 1);
        mbar_init(wqbar, 1);
        mbar_init(qa_local, ET);
        mbar_init(qa_remote, 1);
        mbar_init(q_done, 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(tslot, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;

    if (warp == WP) {
        if (lane == 0) {  // every tile of this CTA at once: nothing is reused
            const CUtensorMap* maps[S::NT] = {&mapWo, &mapWo, &mapW1, &mapW1, &mapW2, &mapW2};
            const int xs[S::NT] = {0, 64, 0, 64, c * S::CH, c * S::CH + 64};
            const int ys[S::NT] = {0, 0, c * S::CH, c * S::CH, 0, 0};
            for (int i = 0; i < S::NT; ++i) {
                mbar_arrive_expect_tx(&full[i], S::TILE);
                tma_load_2d(Wt + i * S::TILE, maps[i], &full[i], xs[i], ys[i]);
            }
            if (NCL > 1) mbar_arrive_expect_tx(rbar, (uint32_t)(NCL - 1) * S::SLICE_BYTES(NCL));
            if (qkv) {
                mbar_arrive_expect_tx(wqbar, 2 * NQ * 128);
                tma_load_2d(Wq, &mapWq, wqbar, 0, c * NQ);
                tma_load_2d(Wq + NQ * 128, &mapWq, wqbar, 64, c * NQ);
                mbar_arrive_expect_tx(qa_remote, (uint32_t)(NCL - 1) * 2 * RW * 128);
            }
            pdl_wait();  // the attention rows are the previous kernel's output
            mbar_arrive_expect_tx(abar, 2 * S::TILE);
            tma_load_2d(A, &mapAtt, abar, 0, m0);
            tma_load_2d(A + S::TILE, &mapAtt, abar, 64, m0);
        }
        __syncwarp();
    } else if (warp == WM) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(128, 128);
            bool ok = true;
            // D (+)= A (two 64-column k-blocks at a_addr) x W tiles i0, i0 + 1
            auto mma_pair = [&](uint32_t a_addr, int i0, uint32_t d_tmem) {
                for (int kb = 0; kb < 2; ++kb) {
                    ok = ok && mbar_wait(&full[i0 + kb], 0, a.err, 61);
                    if (!ok) return;
                    tc_fence_after();
                    const uint32_t b_addr = smem_u32(Wt + (i0 + kb) * S::TILE);
#pragma unroll
                    for (int kk = 0; kk < S::BK / 16; ++kk)
                        tc_mma_bf16(d_tmem, sw128_desc(a_addr + kb * S::TILE + kk * 32),
                                    sw128_desc(b_addr + kk * 32), idesc, (kb | kk) ? 1u : 0u);
                }
            };
            const uint32_t a0 = smem_u32(A), r0 = smem_u32(Rg);
            ok = mbar_wait(abar, 0, a.err, 62);
            tc_fence_after();
            mma_pair(a0, 0, tmem);
            tc_commit(o_done);
            ok = ok && mbar_wait(x1_ready, 0, a.err, 63);
            tc_fence_after();
            mma_pair(a0, 2, tmem + 128);
            tc_commit(h_done);
            ok = ok && mbar_wait(e2_done, 0, a.err, 64);
            tc_fence_after();
            mma_pair(r0, 4, tmem);
            tc_commit(y_done);
        }
        __syncwarp();
    } else {
        // epilogue warps 0-15: row t = 32 (warp % 4) + lane, columns cb..cb+CW-1
        const int tid = threadIdx.x, q = warp & 3, hh = warp >> 2, t = q * 32 + lane, cb = hh * CW;
        const bool live = t < rows;
        {   // parameters, then (after the wait) the residual tile; all loads
            // issued before any store
            const float* src[6] = {a.b_o, a.ln1_g, a.ln1_b, a.b_2, a.ln2_g, a.ln2_b};
            constexpr int NP = (6 * D + ET - 1) / ET;
            float pv[NP];
#pragma unroll
            for (int k = 0; k < NP; ++k) {
                const int i = tid + ET * k;
                pv[k] = i < 6 * D ? src[i / D][i % D] : 0.f;
            }
            const float b1v = tid < S::CH ? a.b_1[c * S::CH + tid] : 0.f;
            pdl_wait();
            constexpr int NV = S::BM * D / 4 / ET;
            float4 v[NV];
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int f = tid + ET * k, r = f >> 5, c4 = f & 31;
                v[k] = r < rows ? *reinterpret_cast<const float4*>(a.x + (size_t)(m0 + r) * D + 4 * c4)
                                : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int k = 0; k < NV; ++k) {
                const int f = tid + ET * k, r = f >> 5, c4 = f & 31;
                *reinterpret_cast<float4*>(res + r * S::RLD + 4 * c4) = v[k];
            }
#pragma unroll
            for (int k = 0; k < NP; ++k)
                if (tid + ET * k < 6 * D) prm[tid + ET * k] = pv[k];
            if (tid < S::CH) prm[6 * D + tid] = b1v;
        }
        epi_sync512();
        const float *p_bo = prm + cb, *p_g1 = prm + D + cb, *p_be1 = prm + 2 * D + cb, *p_b2 = prm + 3 * D + cb;
        const float* p_b1 = prm + 6 * D + cb;
        const uint32_t tl = tmem + ((uint32_t)(q * 32) << 16);
        float* xr = res + t * S::RLD + cb;
        float y[CW];
        mbar_wait(o_done, 0, a.err, 65);
        tc_fence_after();
        tmem_ld32(tl + cb, y);
#pragma unroll
        for (int cc = 0; cc < CW; cc += 4) {
            const float4 r4 = *reinterpret_cast<const float4*>(xr + cc);
            y[cc] += p_bo[cc] + r4.x;
            y[cc + 1] += p_bo[cc + 1] + r4.y;
            y[cc + 2] += p_bo[cc + 2] + r4.z;
            y[cc + 3] += p_bo[cc + 3] + r4.w;
        }
        {   // LN1 (row quarters held by the four warps of lane quarter q)
            float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
            for (int cc = 0; cc < CW; cc += 4) {
                s0 += y[cc];
                s1 += y[cc + 1];
                s2 += y[cc + 2];
                s3 += y[cc + 3];
            }
            red[hh * S::BM + t] = (s0 + s1) + (s2 + s3);
            epi_sync512();
            const float mean = ((red[t] + red[S::BM + t]) + (red[2 * S::BM + t] + red[3 * S::BM + t])) / D;
            s0 = s1 = s2 = s3 = 0.f;
#pragma unroll
            for (int cc = 0; cc < CW; cc += 4) {
                s0 = fmaf(y[cc] - mean, y[cc] - mean, s0);
                s1 = fmaf(y[cc + 1] - mean, y[cc + 1] - mean, s1);
                s2 = fmaf(y[cc + 2] - mean, y[cc + 2] - mean, s2);
                s3 = fmaf(y[cc + 3] - mean, y[cc + 3] - mean, s3);
            }
            red[(4 + hh) * S::BM + t] = (s0 + s1) + (s2 + s3);
            epi_sync512();  // also ends every read of the residual tile
            const float var = ((red[4 * S::BM + t] + red[5 * S::BM + t]) + (red[6 * S::BM + t] + red[7 * S::BM + t])) / D;
            const float inv = 1.0f / sqrtf(var + LN_EPS);
#pragma unroll
            for (int cc = 0; cc < CW; ++cc) y[cc] = live ? (y[cc] - mean) * inv * p_g1[cc] + p_be1[cc] : 0.f;
        }
        tmem_st32(tl + 256 + cb, y);
#pragma unroll
        for (int c0 = 0; c0 < CW; c0 += 16) st_swizzled16(A, t, cb + c0, y + c0);
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(x1_ready);
        // FFN1 chunk c: ReLU(H + b_1) -> bf16 operand of FFN2 (residual region)
        mbar_wait(h_done, 0, a.err, 66);
        tc_fence_after();
        tmem_ld32(tl + 128 + cb, y);
#pragma unroll
        for (int cc = 0; cc < CW; ++cc) y[cc] = fmaxf(y[cc] + p_b1[cc], 0.f);
#pragma unroll
        for (int c0 = 0; c0 < CW; c0 += 16) st_swizzled16(Rg, t, cb + c0, y + c0);
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(e2_done);
        // this CTA's FFN2 partial (CTA 0: + b_2 + x1) into the residual region
        mbar_wait(y_done, 0, a.err, 67);
        tc_fence_after();
        tmem_ld32(tl + cb, y);
        if (c == 0) {
            float x1[CW];
            tmem_ld32(tl + 256 + cb, x1);
#pragma unroll
            for (int cc = 0; cc < CW; ++cc) y[cc] += p_b2[cc] + x1[cc];
        }
#pragma unroll
        for (int cc = 0; cc < CW; cc += 4)
            *reinterpret_cast<float4*>(xr + cc) = make_float4(y[cc], y[cc + 1], y[cc + 2], y[cc + 3]);
        fence_proxy_async_smem();  // the bulk copies below read these writes
    }
    // every partial of the cluster is in shared memory and every CTA's
    // weight region is free
    cluster_sync();
    pdl_trigger();  // the next kernel may be scheduled while the rows are finished
    if (threadIdx.x == 0 && NCL > 1) {  // slice p of this partial -> slot c of CTA p's weight region
        for (int p = 0; p < NCL; ++p)
            if (p != c)
                bulk_s2peer(Wt + (size_t)c * S::SLICE_BYTES(NCL), res + p * (S::BM / NCL) * S::RLD,
                            (uint32_t)S::SLICE_BYTES(NCL), rbar, (uint32_t)p);
        bulk_commit();
    }
    if (warp < S::EW) {
        // rows c RW .. c RW + RW - 1 of the tile: TPR threads per row, CPT columns each
        constexpr int RW = S::BM / NCL, TPR = ET / RW, CPT = D / TPR;
        const int tid = threadIdx.x, rr = tid / TPR, col = (tid % TPR) * CPT, r = c * RW + rr;
        const float *p_g2 = prm + 4 * D, *p_be2 = prm + 5 * D;
        // slice of CTA pr: this CTA's own partial for pr = c, else slot pr
        // of the weight region (all loads before the first sum)
        if (NCL > 1) mbar_wait(rbar, 0, a.err, 68);
        const float* wslots = reinterpret_cast<const float*>(Wt);
        float4 ld[NCL][CPT / 4];
#pragma unroll
        for (int pr = 0; pr < NCL; ++pr) {
            const float* src = pr == c ? res + r * S::RLD + col : wslots + (pr * RW + rr) * S::RLD + col;
#pragma unroll
            for (int j = 0; j < CPT / 4; ++j) ld[pr][j] = *reinterpret_cast<const float4*>(src + 4 * j);
        }
        float v[CPT];
#pragma unroll
        for (int j = 0; j < CPT / 4; ++j) {
            v[4 * j] = ld[0][j].x; v[4 * j + 1] = ld[0][j].y; v[4 * j + 2] = ld[0][j].z; v[4 * j + 3] = ld[0][j].w;
        }
#pragma unroll
        for (int pr = 1; pr < NCL; ++pr)
#pragma unroll
            for (int j = 0; j < CPT / 4; ++j) {
                v[4 * j] += ld[pr][j].x; v[4 * j + 1] += ld[pr][j].y;
                v[4 * j + 2] += ld[pr][j].z; v[4 * j + 3] += ld[pr][j].w;
            }
        // LN2: row sums over the TPR consecutive lanes of the row
        float sm = 0.f;
#pragma unroll
        for (int j = 0; j < CPT; ++j) sm += v[j];
#pragma unroll
        for (int o = TPR >> 1; o > 0; o >>= 1) sm += __shfl_xor_sync(0xffffffffu, sm, o);
        const float mean = sm / D;
        float sq = 0.f;
#pragma unroll
        for (int j = 0; j < CPT; ++j) sq = fmaf(v[j] - mean, v[j] - mean, sq);
#pragma unroll
        for (int o = TPR >> 1; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
        const float inv = 1.0f / sqrtf(sq / D + LN_EPS);
        if (qkv) {  // this row slice of the next layer's A tile (zeros past the rows)
            float o[CPT];
#pragma unroll
            for (int j = 0; j < CPT; ++j)
                o[j] = r < rows ? (v[j] - mean) * inv * p_g2[col + j] + p_be2[col + j] : 0.f;
            if constexpr (CPT == 16) st_swizzled16(A, r, col, o);
            else if constexpr (CPT == 8) st_swizzled8(A, r, col, o);
            else if constexpr (CPT == 4) st_swizzled4(A, r, col, o);
            fence_proxy_async_smem();
            mbar_arrive(qa_local);
        }
        if (r < rows) {
            float* xo = a.x + (size_t)(m0 + r) * D + col;
            bf16* xbo = a.xb + (size_t)(m0 + r) * D + col;
#pragma unroll
            for (int j = 0; j < CPT; j += 4) {
                float4 o;
                o.x = (v[j] - mean) * inv * p_g2[col + j] + p_be2[col + j];
                o.y = (v[j + 1] - mean) * inv * p_g2[col + j + 1] + p_be2[col + j + 1];
                o.z = (v[j + 2] - mean) * inv * p_g2[col + j + 2] + p_be2[col + j + 2];
                o.w = (v[j + 3] - mean) * inv * p_g2[col + j + 3] + p_be2[col + j + 3];
                *reinterpret_cast<float4*>(xo + j) = o;
                const __nv_bfloat162 p0 = __floats2bfloat162_rn(o.x, o.y);
                const __nv_bfloat162 p1 = __floats2bfloat162_rn(o.z, o.w);
                uint2 w;
                w.x = *reinterpret_cast<const uint32_t*>(&p0);
                w.y = *reinterpret_cast<const uint32_t*>(&p1);
                *reinterpret_cast<uint2*>(xbo + j) = w;
            }
        }
    }
    if (qkv) {
        if (threadIdx.x == 0) {  // this CTA's finished rows -> the same rows of every peer's A tile
            mbar_wait(qa_local, 0, a.err, 69);
            for (int p = 0; p < NCL; ++p)
                if (p != c)
                    for (int kb = 0; kb < 2; ++kb) {
                        unsigned char* blk = A + kb * S::TILE + c * RW * 128;
                        bulk_s2peer(blk, blk, (uint32_t)(RW * 128), qa_remote, (uint32_t)p);
                    }
            bulk_commit();
        } else if (warp == WM && lane == 0) {
            bool ok = mbar_wait(wqbar, 0, a.err, 70);
            ok = ok && mbar_wait(qa_local, 0, a.err, 71);
            ok = ok && mbar_wait(qa_remote, 0, a.err, 72);
            tc_fence_after();
            if (ok) {
                const uint32_t idesc = idesc_bf16(128, NQ), a0 = smem_u32(A), q0 = smem_u32(Wq);
                for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                    for (int kk = 0; kk < S::BK / 16; ++kk)
                        tc_mma_bf16(tmem + 384, sw128_desc(a0 + kb * S::TILE + kk * 32),
                                    sw128_desc(q0 + kb * NQ * 128 + kk * 32), idesc, (kb | kk) ? 1u : 0u);
            }
            tc_commit(q_done);
        }
        __syncwarp();
        if (warp < 8) {
            // rows t = 32 (warp % 4) + lane; the column halves of the slice by
            // warps 0-3 / 4-7 when they split into 16-column groups (warps
            // 8-15 have no part here)
            constexpr int HALF = (NQ / 2) % 16 == 0 ? NQ / 2 : NQ;
            const int q = warp & 3, hh = warp >> 2, t = q * 32 + lane, r = m0 + t;
            const bool ok = mbar_wait(q_done, 0, a.err, 73);
            tc_fence_after();
            const bool mine = HALF == NQ ? hh == 0 : true;
            const int s = t < rows ? a.row_seq[r] : -1, pos = t < rows ? a.row_pos[r] : 0;
            const uint32_t tl = tmem + ((uint32_t)(q * 32) << 16) + 384;
            for (int c0 = hh * HALF; mine && c0 < hh * HALF + HALF; c0 += 16) {
                float v[16];
                tmem_ld16(tl + c0, v);
                if (!ok || t >= rows) continue;
                const int col = c * NQ + c0, which = col / D, cc = col - which * D;
#pragma unroll
                for (int i = 0; i < 16; ++i) v[i] += a.b_qkv[col + i];
                if (which == 0) {
                    st_bf16x16(a.q_out + (size_t)r * D + cc, v);
                } else if (s >= 0) {
                    const int h = cc / a.dh, e = cc - h * a.dh;
                    const size_t o = ((((size_t)a.layer * a.Bmax + s) * a.nh + h) * (size_t)a.n_max + pos) * a.dh + e;
                    if (which == 2 && a.v_f16) st_f16x16_of_bf16(a.vc + o, v);
                    else st_bf16x16((which == 1 ? a.kc : a.vc) + o, v);
                }
            }
        }
    }
    // the sources of this CTA's bulk copies have been read before it exits;
    // its own slots were all filled (rbar, qa_remote) before they were read
    if (threadIdx.x == 0 && (NCL > 1 || qkv)) bulk_wait_read_all();
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 512);
    pdl_trigger();
}

int mlp_cl_supported(int d, int F) {
    const int n = F / MlpClShape::CH;
    return d == MlpClShape::D && F % MlpClShape::CH == 0 && (n == 1 || n == 2 || n == 4 || n == 8);
}

template <int NCL>
static cudaError_t launch_mlp_ncl(const CUtensorMap& att, const CUtensorMap& wo, const CUtensorMap& w1,
                                  const CUtensorMap& w2, const CUtensorMap& wq, const MlpArgs& a, cudaStream_t st) {
    const size_t sm = MlpClShape::SMEM;
    cudaError_t e = cudaFuncSetAttribute(k_mlp_cl<NCL>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    const int ncl = NCL;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(ncl, (a.R + 127) / 128, 1);
    cfg.blockDim = dim3(MlpClShape::THREADS, 1, 1);
    cfg.dynamicSmemBytes = sm;
    cfg.stream = st;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = ncl;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = g_pdl ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, k_mlp_cl<NCL>, att, wo, w1, w2, wq, a);
}

int mlp_cl_qkv_cols(int d, int F) {
    if (!mlp_cl_supported(d, F)) return 0;
    const int n = F / MlpClShape::CH;
    return MlpClShape::QKV_OK(n) ? MlpClShape::NQ(n) : 0;
}

cudaError_t launch_mlp_cl(const CUtensorMap& att, const CUtensorMap& wo, const CUtensorMap& w1,
                          const CUtensorMap& w2, const CUtensorMap& wq, const MlpArgs& a, cudaStream_t st) {
    if (a.R <= 0) return cudaSuccess;
    if (!mlp_cl_supported(MlpClShape::D, a.F)) return cudaErrorInvalidValue;
    if (a.qkv && !mlp_cl_qkv_cols(MlpClShape::D, a.F)) return cudaErrorInvalidValue;
    switch (a.F / MlpClShape::CH) {
        case 1: return launch_mlp_ncl<1>(att, wo, w1, w2, wq, a, st);
        case 2: return launch_mlp_ncl<2>(att, wo, w1, w2, wq, a, st);
        case 4: return launch_mlp_ncl<4>(att, wo, w1, w2, wq, a, st);
        case 8: return launch_mlp_ncl<8>(att, wo, w1, w2, wq, a, st);
    }
    return cudaErrorInvalidValue;
}

int mlp_tc_supported(int d, int F) { return d == MlpShape::D && F % MlpShape::CH == 0 && F <= MlpShape::PF; }

cudaError_t launch_mlp_tc(const CUtensorMap& att, const CUtensorMap& wo, const CUtensorMap& w1,
                          const CUtensorMap& w2, const MlpArgs& a, cudaStream_t st) {
    if (a.R <= 0) return cudaSuccess;
    if (!mlp_tc_supported(MlpShape::D, a.F)) return cudaErrorInvalidValue;
    const size_t sm = MlpShape::SMEM;
    cudaError_t e = cudaFuncSetAttribute(k_mlp_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    return launch_k(k_mlp_tc, dim3((a.R + 127) / 128), dim3(320), sm, st, att, wo, w1, w2, a);
}

}  // namespace tppsd
