// Causal attention of the target model for bf16 caches (verify pass: gamma+1
// queries per sequence; AR step: 1 query; prefill: chunks of 16 queries).
//
// CTA = (up to 16 query rows of one sequence, one head), four warps.  The
// K and V of one (sequence, layer, head) are contiguous [position][d_head]
// in HBM, so every key tile is one copy into the warp's own double-buffered
// shared stage, completing on an mbarrier: a TMA tensor-map box with the
// row-width swizzle for d_head >= 32 (conflict-free ldmatrix over
// consecutive keys), a linear bulk copy (cp.async.bulk) for d_head 16.  The
// keys 0..maxpos are cut into four contiguous ranges of equal length (a
// multiple of 8 keys), one per warp, so all four warps work even when the
// context is a single tile; each warp keeps its own online-softmax state
// (flash-decoding split inside the CTA).  S = Q K^T uses mma.sync
// m16n8k16 with bf16 inputs (exact products, fp32 accumulation); P V splits
// P into two bf16 parts (P = P_hi + P_lo, 16 significant bits) against the
// bf16 V tile as copied, with fp32 accumulation.  The online softmax's
// exponentials use the ex2.approx instruction (PTX ISA: relative error
// about 2^-22), in log2 units.  The four partial results
// are merged through shared memory, each written over its warp's own stages.
// Two tile sizes: 1 KB tiles keep a CTA at ~17 KB of shared memory and 72
// registers per thread (d_head <= 32), so seven CTAs fit an SM and a grid of
// up to 7 x (SM count) items (the 1 024 (sequence, head) items of a
// 256-sequence verify pass) runs in one wave; larger grids run in several
// waves anyway and take 2 KB tiles (half the tiles per key range).
#include <stdlib.h>

#include "common.cuh"
#include "engine.h"
#include "tc_ptx.cuh"

namespace tppsd {

template <int DH, int TB>
struct AttnShape {
    // keys per tile: TB bytes of K and TB of V (at least 16 keys, one P V step)
    static constexpr int KT = TB / (2 * DH) < 16 ? 16 : TB / (2 * DH);
    static constexpr int TILE_BYTES = KT * DH * 2;
    static constexpr int STAGE_BYTES = 2 * TILE_BYTES;
    // warp w's two stages at (2w + s) STAGE_BYTES from a 1024-byte aligned
    // base (the swizzle pattern of a tile repeats within 1 KB), then the
    // eight mbarriers and the row positions
    static constexpr int WARP_BYTES = 2 * STAGE_BYTES;
    static constexpr int OFF_BAR = 4 * WARP_BYTES;
    // a warp's partial result (max, sum, 16 x DH numerators), written over
    // its own stages once its last tile is consumed
    static constexpr int MERGE_FLOATS = 16 * DH + 32;
    static_assert(MERGE_FLOATS * 4 <= 2 * STAGE_BYTES, "partial result must fit the warp's stages");
    static_assert(TILE_BYTES % 1024 == 0 || DH < 32, "swizzled tiles start on 1 KB boundaries");
    static constexpr int SMEM = OFF_BAR + 64 + 16 * 4 + 1024;
    // d_head >= 32: tiles by TMA tensor maps with the row-width swizzle (32,
    // 64 or 128 bytes, 16-byte chunk c of row r at c ^ ((r * rowb) >> 7)),
    // so ldmatrix phases over consecutive keys meet no bank conflicts;
    // d_head = 16 keeps linear bulk copies
    static constexpr bool TMA = DH >= 32;
};

// Byte offset of 16-byte chunk c of row r of a tile of DH-wide bf16 rows
// as the tensor map's swizzle lays it out (linear when not swizzled).
template <int DH, bool SWZ>
__device__ __forceinline__ uint32_t tile_off(int r, int c) {
    constexpr int ROWB = DH * 2, MASK = ROWB == 128 ? 7 : ROWB == 64 ? 3 : 1;
    return SWZ ? (uint32_t)(r * ROWB + ((c ^ (((r * ROWB) >> 7) & MASK)) << 4)) : (uint32_t)(r * ROWB + (c << 4));
}

__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// 2^x by the hardware approximation (x = -inf gives +0)
__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2(uint32_t (&r)[2], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];" : "=r"(r[0]), "=r"(r[1]) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_trans(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
__device__ __forceinline__ void split_bf16x2(float x, float y, uint32_t& hi, uint32_t& lo) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
    const float2 hf = __bfloat1622float2(h);
    const __nv_bfloat162 l = __floats2bfloat162_rn(x - hf.x, y - hf.y);
    hi = *reinterpret_cast<const uint32_t*>(&h);
    lo = *reinterpret_cast<const uint32_t*>(&l);
}

// TB = 1024: small footprint, seven CTAs per SM (d_head <= 32); TB = 2048:
// fewer tiles per key range, four CTAs per SM.
template <int DH, int TB>
__global__ void __launch_bounds__(128, (DH >= 64 || TB > 1024) ? 4 : 7)
    k_attn_mma(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap, AttArgs<bf16> a,
               int* err) {
    using S = AttnShape<DH, TB>;
    constexpr int KT = S::KT, NT = KT / 8, KS = DH / 16;
    pdl_wait();
    extern __shared__ __align__(128) unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, t4 = lane & 3;
    const int h = blockIdx.y;
    const int seq = a.g0 / a.q_per_seq + blockIdx.z;
    const int r_lo = max(0, seq * a.q_per_seq - a.g0);
    const int r_hi = min(a.count, (seq + 1) * a.q_per_seq - a.g0);
    const int rb = r_lo + blockIdx.x * 16;
    const int re = min(rb + 16, r_hi);
    if (rb >= re) return;
    const int s = a.row_seq[rb];
    const int maxpos = a.row_pos[re - 1];  // rows of a sequence are in position order
    if (s < 0) return;  // rows of one sequence are all active or all inactive
    const int nq = re - rb;
    unsigned char* wbase = smem + warp * S::WARP_BYTES;
    uint64_t* bars = (uint64_t*)(smem + S::OFF_BAR) + 2 * warp;
    int* qpos = (int*)(smem + S::OFF_BAR + 64);
    // this warp's key range [klo, khi)
    const int nkeys = maxpos + 1;
    const int share = (((nkeys + 3) / 4) + 7) & ~7;
    const int klo = min(nkeys, warp * share), khi = min(nkeys, klo + share);
    const int ntl = (khi - klo + KT - 1) / KT;
    const long long yrow = (((long long)a.layer * a.kv.Bmax + s) * a.nh + h) * a.kv.n_max;  // tensor-map row of key 0
    const bf16* kg = a.kc + (size_t)yrow * DH;
    const bf16* vg = a.vc + (size_t)yrow * DH;
    auto issue = [&](int tile, int stage) {
        const int k0 = klo + tile * KT, cnt = min(KT, khi - k0);
        unsigned char* st = wbase + stage * S::STAGE_BYTES;
        if constexpr (S::TMA) {  // whole boxes: keys past the range are masked, V rows zeroed
            mbar_arrive_expect_tx(&bars[stage], 2 * S::TILE_BYTES);
            tma_load_2d(st, &kmap, &bars[stage], 0, (int)(yrow + k0));
            tma_load_2d(st + S::TILE_BYTES, &vmap, &bars[stage], 0, (int)(yrow + k0));
        } else {
            const uint32_t bytes = (uint32_t)cnt * DH * 2;
            mbar_arrive_expect_tx(&bars[stage], 2 * bytes);
            bulk_load(st, kg + (size_t)k0 * DH, bytes, &bars[stage]);
            bulk_load(st + S::TILE_BYTES, vg + (size_t)k0 * DH, bytes, &bars[stage]);
        }
    };
    // the first tile's copy is in flight before anything else is loaded
    if (lane == 0) {
        mbar_init(&bars[0], 1);
        mbar_init(&bars[1], 1);
        mbar_fence_init();
        if (ntl > 0) issue(0, 0);
    }
    if (threadIdx.x < 16) qpos[threadIdx.x] = threadIdx.x < nq ? a.row_pos[rb + threadIdx.x] : -1;

    // Q fragments (rows g and g+8 of this CTA, all DH columns), bf16 pairs
    uint32_t qa[KS][4];
#pragma unroll
    for (int k = 0; k < KS; ++k) {
        const int c0 = 16 * k + 2 * t4;
        auto ld = [&](int row, int col) -> uint32_t {
            if (row >= nq) return 0u;
            return *reinterpret_cast<const uint32_t*>(a.q + (size_t)(rb + row) * a.d + h * DH + col);
        };
        qa[k][0] = ld(g, c0);
        qa[k][1] = ld(g + 8, c0);
        qa[k][2] = ld(g, c0 + 8);
        qa[k][3] = ld(g + 8, c0 + 8);
    }
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;  // rows g, g+8
    float o[DH / 8][4];
#pragma unroll
    for (int n = 0; n < DH / 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;

    __syncthreads();  // qpos and the mbarrier inits are visible
    const int pos_g = qpos[g], pos_g8 = qpos[g + 8];  // -1 for padding rows
    const int pos_first = qpos[0];                    // the smallest position of the rows
    const float scale2 = a.scale * 1.4426950408889634f;  // scores in log2 units: exp2 below
    bool ok = true;
    for (int it = 0; it < ntl && ok; ++it) {
        const int stage = it & 1;
        if (lane == 0 && it + 1 < ntl) issue(it + 1, stage ^ 1);
        ok = __all_sync(0xffffffffu, mbar_wait(&bars[stage], (it >> 1) & 1, err, 21));
        if (!ok) break;
        unsigned char* st = wbase + stage * S::STAGE_BYTES;
        const bf16* ks = (const bf16*)st;
        const bf16* vs = (const bf16*)(st + S::TILE_BYTES);
        const int k0 = klo + it * KT, cnt = min(KT, khi - k0);
        if (cnt < KT) {  // V rows past the range -> 0 (their P is 0, and 0 * NaN bits is NaN)
            for (int i = cnt * DH / 8 + lane; i < KT * DH / 8; i += 32)
                reinterpret_cast<uint4*>(const_cast<bf16*>(vs))[i] = make_uint4(0, 0, 0, 0);
            fence_proxy_async_smem();  // before the stage is refilled by the async proxy
            __syncwarp();
        }
        // S = Q K^T for KT keys; K fragments by ldmatrix (8 keys x 8 dims a
        // matrix; keys past the copied ones read stale rows, masked below)
        float sc[NT][4];
        const uint32_t kbase = smem_u32(ks);
#pragma unroll
        for (int n = 0; n < NT; ++n) {
            sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
            for (int k = 0; k + 1 < KS; k += 2) {  // two k-steps (32 dims) per x4
                uint32_t b[4];
                ldsm_x4(b, kbase + tile_off<DH, S::TMA>(8 * n + (lane & 7), 2 * k + (lane >> 3)));
                mma_bf16(sc[n], qa[k], b[0], b[1]);
                mma_bf16(sc[n], qa[k + 1], b[2], b[3]);
            }
            if constexpr (KS % 2) {
                uint32_t b[2];
                ldsm_x2(b, kbase + tile_off<DH, S::TMA>(8 * n + (lane & 7), 2 * (KS - 1) + ((lane >> 3) & 1)));
                mma_bf16(sc[n], qa[KS - 1], b[0], b[1]);
            }
        }
        // scale, mask (keys past the copied ones, and causal: only tiles that
        // reach past the first row's position need it), online softmax in
        // log2 units (rows g and g+8; quad reductions)
        float mx0 = -INFINITY, mx1 = -INFINITY;
        if (cnt == KT && k0 + KT - 1 <= pos_first) {
#pragma unroll
            for (int n = 0; n < NT; ++n) {
#pragma unroll
                for (int e = 0; e < 4; ++e) sc[n][e] *= scale2;
                mx0 = fmaxf(mx0, fmaxf(sc[n][0], sc[n][1]));
                mx1 = fmaxf(mx1, fmaxf(sc[n][2], sc[n][3]));
            }
        } else {
#pragma unroll
            for (int n = 0; n < NT; ++n) {
                const int kt = 8 * n + 2 * t4, key = k0 + kt;
                const bool in0 = kt < cnt, in1 = kt + 1 < cnt;
                sc[n][0] = (in0 && key <= pos_g) ? sc[n][0] * scale2 : -INFINITY;
                sc[n][1] = (in1 && key + 1 <= pos_g) ? sc[n][1] * scale2 : -INFINITY;
                sc[n][2] = (in0 && key <= pos_g8) ? sc[n][2] * scale2 : -INFINITY;
                sc[n][3] = (in1 && key + 1 <= pos_g8) ? sc[n][3] * scale2 : -INFINITY;
                mx0 = fmaxf(mx0, fmaxf(sc[n][0], sc[n][1]));
                mx1 = fmaxf(mx1, fmaxf(sc[n][2], sc[n][3]));
            }
        }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
        const float ref0 = mn0 == -INFINITY ? 0.f : mn0, ref1 = mn1 == -INFINITY ? 0.f : mn1;
        const float c0 = ex2_approx(m0 - ref0), c1 = ex2_approx(m1 - ref1);
        float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
        for (int n = 0; n < NT; ++n) {
            sc[n][0] = ex2_approx(sc[n][0] - ref0);
            sc[n][1] = ex2_approx(sc[n][1] - ref0);
            sc[n][2] = ex2_approx(sc[n][2] - ref1);
            sc[n][3] = ex2_approx(sc[n][3] - ref1);
            rs0 += sc[n][0] + sc[n][1];
            rs1 += sc[n][2] + sc[n][3];
        }
        rs0 += __shfl_xor_sync(0xffffffffu, rs0, 1);
        rs0 += __shfl_xor_sync(0xffffffffu, rs0, 2);
        rs1 += __shfl_xor_sync(0xffffffffu, rs1, 1);
        rs1 += __shfl_xor_sync(0xffffffffu, rs1, 2);
        l0 = l0 * c0 + rs0;
        l1 = l1 * c1 + rs1;
        m0 = mn0;
        m1 = mn1;
#pragma unroll
        for (int n = 0; n < DH / 8; ++n) {
            o[n][0] *= c0; o[n][1] *= c0;
            o[n][2] *= c1; o[n][3] *= c1;
        }
        // O += P V with P = P_hi + P_lo (two bf16 parts) and bf16 V fragments by
        // ldmatrix.trans; keys past the copied ones have P = 0 (V there is masked)
        const uint32_t vbase = smem_u32(vs);
#pragma unroll
        for (int kk = 0; kk < KT / 16; ++kk) {
            uint32_t ph[4], pl[4];
            split_bf16x2(sc[2 * kk][0], sc[2 * kk][1], ph[0], pl[0]);
            split_bf16x2(sc[2 * kk][2], sc[2 * kk][3], ph[1], pl[1]);
            split_bf16x2(sc[2 * kk + 1][0], sc[2 * kk + 1][1], ph[2], pl[2]);
            split_bf16x2(sc[2 * kk + 1][2], sc[2 * kk + 1][3], ph[3], pl[3]);
#pragma unroll
            for (int n = 0; n < DH / 8; n += 2) {
                const int key = 16 * kk + (lane & 15);
                const int col = 8 * n + (lane >> 4) * 8;
                uint32_t vb[4];
                ldsm_x4_trans(vb, vbase + tile_off<DH, S::TMA>(key, col >> 3));
                mma_bf16(o[n], ph, vb[0], vb[1]);
                mma_bf16(o[n], pl, vb[0], vb[1]);
                mma_bf16(o[n + 1], ph, vb[2], vb[3]);
                mma_bf16(o[n + 1], pl, vb[2], vb[3]);
            }
        }
        __syncwarp();
    }
    pdl_trigger();  // the next kernel may be scheduled while the partials are merged
    // per-warp partial results -> shared memory (over this warp's stages)
    auto mslot = [&](int w) { return (float*)(smem + w * S::WARP_BYTES); };
    float* mw = mslot(warp);
    if (t4 == 0) {
        mw[g] = m0; mw[g + 8] = m1;
        mw[16 + g] = l0; mw[16 + g + 8] = l1;
    }
#pragma unroll
    for (int n = 0; n < DH / 8; ++n) {
        const int col = 8 * n + 2 * t4;
        mw[32 + g * DH + col] = o[n][0];
        mw[32 + g * DH + col + 1] = o[n][1];
        mw[32 + (g + 8) * DH + col] = o[n][2];
        mw[32 + (g + 8) * DH + col + 1] = o[n][3];
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nq * DH; i += blockDim.x) {
        const int row = i / DH, col = i % DH;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < 4; ++w) M = fmaxf(M, mslot(w)[row]);
        float L = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            const float* p = mslot(w);
            if (p[row] == -INFINITY) continue;
            const float e = exp2f(p[row] - M);
            L += p[16 + row] * e;
            O += p[32 + row * DH + col] * e;
        }
        if (a.attnhp) {  // a = sum f v / (1 + sum f); h <- h + tanh(a)
            const size_t xi = (size_t)(rb + row) * a.d + h * DH + col;
            const float hn = a.x[xi] + tanhf(O / (L + exp2f(-M)));  // exp(-m) in log2 units
            a.x[xi] = hn;
            a.hb[(size_t)(rb + row) * 2 * a.d + a.d + h * DH + col] = __float2bfloat16_rn(hn);
        } else {
            a.out[(size_t)(rb + row) * a.d + h * DH + col] = __float2bfloat16_rn(O / L);
        }
    }
    pdl_trigger();
}

template <int DH, int TB>
static cudaError_t launch_attn_t(const AttArgs<bf16>& a, dim3 grid, int* err, cudaStream_t st) {
    using S = AttnShape<DH, TB>;
    const int sm = S::SMEM;
    cudaFuncSetAttribute(k_attn_mma<DH, TB>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
    CUtensorMap mk{}, mv{};
    if (S::TMA) {
        // the caches of layers 0..layer as [(layer, sequence, head, position)][d_head]
        const long long items = (long long)(a.layer + 1) * a.kv.Bmax * a.nh;
        if (!kv_tile_map(&mk, a.kc, DH, a.kv.n_max, items, S::KT) || !kv_tile_map(&mv, a.vc, DH, a.kv.n_max, items, S::KT))
            return cudaErrorInvalidValue;
    }
    return launch_k(k_attn_mma<DH, TB>, grid, dim3(128), sm, st, mk, mv, a, err);
}

cudaError_t launch_attn_mma(const AttArgs<bf16>& a, int dh, int nh, int nseg, int* err, cudaStream_t st) {
    const dim3 grid((a.q_per_seq + 15) / 16, nh, nseg);
    // small tiles when the grid fits one wave of seven CTAs per SM
    // (TPPSD_ATTN_TILE=1024 / 2048 forces a size)
    static int n_sm = 0;
    if (!n_sm) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n_sm <= 0) n_sm = 148;
    }
    bool small = (long long)grid.x * grid.y * grid.z <= 7LL * n_sm;
    if (const char* f = getenv("TPPSD_ATTN_TILE")) small = atoi(f) == 1024;
    cudaError_t e;
    switch (dh) {
        case 16: e = small ? launch_attn_t<16, 1024>(a, grid, err, st) : launch_attn_t<16, 2048>(a, grid, err, st); break;
        case 32: e = small ? launch_attn_t<32, 1024>(a, grid, err, st) : launch_attn_t<32, 2048>(a, grid, err, st); break;
        case 64: e = launch_attn_t<64, 2048>(a, grid, err, st); break;
        default: return cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tppsd
