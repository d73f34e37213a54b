// Causal attention of the target model on the 5th-generation tensor cores
// (bf16 caches): the verify pass (gamma + 1 queries per sequence, Sec. 4.3
// "Verification"), the AR step (1 query) and prefill / scoring (blocks of
// queries of one sequence).
//
// The keys sit on the M side of both products, so a CTA of four warps owns
// a tile of 128 keys with one TMEM lane (one thread) per key:
//
//   S^T [128 keys][32 queries] = K_tile [128][dh] . Q [32][dh]^T
//   O^T [dh][32]               = V_tile^T [dh][128] . P^T [128][32]
//
// K, V and Q tiles arrive by TMA (cp.async.bulk.tensor) through tensor maps
// over the KV cache (2-D views [rows of (layer, sequence, head, position)]
// [dh]) and the Q rows, in the swizzle the tcgen05 shared-memory
// descriptors read (rows of 2 dh bytes: 64- or 128-byte swizzle).  Per
// tile: S^T goes to TMEM; the softmax reads it back with tcgen05.ld
// (thread = key), takes the tile's per-query maximum (a transposing warp
// butterfly, then the four warps through shared memory), and writes
// P^T = P_hi + P_lo (two bf16 parts, 16 significant bits of P) into shared
// memory as the B operand of the second product (P_hi over the consumed K
// tile); V is the A operand read in MN-major form straight from its TMA
// tile (its M extent beyond dh reads shifted rows that give O^T rows which
// are never used).  O^T of the tile lands in its own TMEM columns, and the
// tiles are merged in registers (running maximum, sum and output, the
// online-softmax recurrence applied once per 128 keys).  The K / V tiles of
// the next STAGES - 1 tiles are in flight while one is processed.  A key
// range longer than the GPU can cover in one wave of CTAs is cut into
// splits (flash-decoding), each CTA writing a partial (max, sum, output)
// and the last CTA of an item, found by an arrival counter, merging them.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>
#include <stdlib.h>

#include "common.cuh"
#include "engine.h"
#include "tc_ptx.cuh"

namespace tppsd {

// Shared-memory layout of one CTA: NSTG stages of (V tile, K tile with P^T
// written over it once S^T is computed), the Q tile, reduction buffers and
// mbarriers.  Tile bases are 1024-byte aligned (the swizzle atoms repeat
// every 512 / 1024 bytes).
template <int DH>
struct AttTcShape {
    static constexpr int NQ = 32;                // query columns of both products
    static constexpr int NSTG = DH == 32 ? 3 : 2;  // K / V stages in flight
    static constexpr int ROWB = DH * 2;          // bytes of one K / V / Q row
    static constexpr int TILE = 128 * ROWB;      // one K or V tile (128 keys)
    static constexpr int PROW = NQ * 2;          // bytes of one P^T row (one key)
    static constexpr int PT = 128 * PROW;        // P^T of a tile (bf16)
    static_assert(PT <= TILE, "P^T is written over the consumed K tile");
    static constexpr int STAGE = 2 * TILE;       // V, then K (P^T)
    static constexpr int V_OFF = 0, K_OFF = TILE;
    static constexpr int OFF_Q = NSTG * STAGE;
    static constexpr int Q_BYTES = ((NQ * ROWB) + 1023) & ~1023;
    // floats: reduction scratch [2][4][32], segment references [2][32], the
    // running output's reference [32], final reference and sum [2][32], and
    // the tiles' segment records (ints)
    static constexpr int OFF_RED = OFF_Q + Q_BYTES;
    static constexpr int OFF_BAR = OFF_RED + (416 + 8) * 4;
    // mbarriers: q, k[NSTG], v[NSTG], pready[NSTG], stfree[NSTG], s[2],
    // ofull[2] (a segment's accumulation complete), oempty[2] (folded)
    static constexpr int NBAR = 1 + 4 * NSTG + 6;
    static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;         // tmem slot, flag
    static constexpr int SMEM = OFF_MISC + 16 + 1024;           // + alignment slack
    static constexpr int TCOLS = 128;  // S^T of two tiles, O^T of two tiles: 32 columns each
    static_assert(TILE % 1024 == 0 && STAGE % 1024 == 0, "tile bases stay 1024-byte aligned");
};

// Layout code of the tcgen05 shared-memory descriptor for rows of `bytes`
// (64- or 128-byte swizzle).
__host__ __device__ constexpr int swz_layout(int bytes) { return bytes == 128 ? 2 : 4; }

__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo, int layout) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFF) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFF) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)layout << 61;
    return d;
}

// Byte offset of 16-byte chunk c of row r in a tile of 64-byte rows, as the
// 64-byte swizzle places it (chunk index XOR address bits 7-8).
__device__ __forceinline__ uint32_t swz64_off(int r, int c) {
    return (uint32_t)(r * 64 + ((c ^ ((r >> 1) & 3)) << 4));
}

template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, float (&v)[N]) {
    static_assert(N == 16 || N == 32, "16 or 32 columns");
    float a[16];
    tmem_ld16(taddr, a);
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = a[i];
    if constexpr (N == 32) {
        tmem_ld16(taddr + 16, a);
#pragma unroll
        for (int i = 0; i < 16; ++i) v[16 + i] = a[i];
    }
}

// Per-warp part of a reduction of QV values per thread over the CTA: a
// transposing butterfly leaves lane l holding the warp's result for query
// q(l), which it writes to red[warp][q].  After a barrier every thread can
// read the four warps' values (warp_red_read).
template <int QV, bool MAX>
__device__ __forceinline__ void warp_red_write(const float (&v)[QV], float* red, int warp, int lane) {
    float w[QV];
#pragma unroll
    for (int i = 0; i < QV; ++i) w[i] = v[i];
    int cnt = QV;
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
        if (cnt > 1) {
            const int half = cnt / 2;
            const bool up = (lane & off) != 0;
#pragma unroll
            for (int i = 0; i < QV / 2; ++i) {
                if (i < half) {
                    const float send = up ? w[i] : w[i + half];
                    const float keep = up ? w[i + half] : w[i];
                    const float got = __shfl_xor_sync(0xffffffffu, send, off);
                    w[i] = MAX ? fmaxf(keep, got) : keep + got;
                }
            }
            cnt = half;
        } else {
            const float got = __shfl_xor_sync(0xffffffffu, w[0], off);
            w[0] = MAX ? fmaxf(w[0], got) : w[0] + got;
        }
    }
    int q;  // the bits of the rounds that halved the set
    if constexpr (QV == 32) q = lane;
    else if constexpr (QV == 16) q = (lane >> 1) & 15;
    else q = 0;
    const bool writer = QV == 32 || (QV == 16 && (lane & 1) == 0) || (QV == 1 && lane == 0);
    if (writer) red[warp * 32 + q] = w[0];
}
template <bool MAX>
__device__ __forceinline__ float warp_red_read(const float* red, int q) {
    const float a = red[q], b = red[32 + q], c = red[64 + q], d = red[96 + q];
    return MAX ? fmaxf(fmaxf(a, b), fmaxf(c, d)) : (a + b) + (c + d);
}


// Named barrier among the `n` threads of warps 0 .. n/32 - 1.
__device__ __forceinline__ void named_sync(int id, int n) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
// The same barrier, returning the AND of every participant's `in`.
__device__ __forceinline__ bool named_sync_and(int id, int n, bool in) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 q, %1, 0;\n\t"
        "bar.red.and.pred p, %2, %3, q;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)in), "r"(id), "r"(n)
        : "memory");
    return r != 0;
}

// The same barrier, returning the OR of every participant's `in`.
__device__ __forceinline__ bool named_sync_or(int id, int n, bool in) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 q, %1, 0;\n\t"
        "bar.red.or.pred p, %2, %3, q;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)in), "r"(id), "r"(n)
        : "memory");
    return r != 0;
}

// Instruction descriptor: kind::f16 with fp16 A/B, fp32 D, both MN-major.
__host__ __device__ constexpr uint32_t idesc_f16_mn(int M, int N) {
    return (1u << 4) | (1u << 15) | (1u << 16) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// QV: the query rows a CTA owns (32, 16, or 1 for one-query passes); the
// softmax evaluates the first nq <= QV of them, and the columns past nq of
// both products hold P = 0.
//
// Warp roles: warps 0-3 own TMEM lane quarters (one key per thread) and run
// the softmax of every tile; warps 0 .. DH/32 - 1 also fold finished O^T
// accumulators into the running result; warp 4 (one thread) issues the TMA
// copies and the MMAs.  Per tile t (smem stage t % NSTG, S^T buffer t % 2):
//   K, V land (kfull, vfull) -> S^T MMA (sfull) -> softmax writes P^T over
//   K (pready) -> O^T MMA accumulates (stfree when the stage may be refilled
//   with tile t + NSTG).
// S^T of tile t + 1 is computed while the softmax of tile t runs, and the
// copies of the next NSTG - 1 tiles are in flight.
//
// Softmax reference: each query keeps a reference m (base-2 units, scores
// scaled by log2(e) / sqrt(d_head)) and every tile's weights are
// P = 2^(s - m), so the O^T MMAs of consecutive tiles accumulate in one TMEM
// buffer with no rescaling and no per-tile reduction across warps.  The
// first tile sets m to its per-query maximum; a later tile whose scores
// exceed m + slack (slack = 15, so that P < 2^15 stays inside fp16) raises m
// to the new maximum, rescales the threads' partial sums, and starts a new
// accumulation segment in the other O^T buffer, while the finished segment
// is folded into the running output (scaled by 2^(m_old - m_new)).
//
// Precision: V is stored in fp16 (the bf16-rounded values, exact in the fp16
// range) and P is rounded to fp16 (11 significant bits); the row sums add
// the same rounded weights, so O^T / sum is an exact weighted mean of V with
// weights within 2^-12 of the softmax's.
template <int DH, int QV>
__global__ void __launch_bounds__(160, 3)
    k_attn_tc(const __grid_constant__ CUtensorMap mapK, const __grid_constant__ CUtensorMap mapV,
              const __grid_constant__ CUtensorMap mapQ, AttTcArgs a) {
    using S = AttTcShape<DH>;
    constexpr int NQ = S::NQ, ROWB = S::ROWB, NSTG = S::NSTG;
    constexpr int LC = QV <= 16 ? 16 : 32;  // TMEM columns read back per tile
    constexpr int LAY_KV = swz_layout(ROWB), LAY_P = swz_layout(S::PROW);
    constexpr uint32_t SBO_KV = 8 * ROWB, SBO_P = 8 * S::PROW;
    constexpr int NMW = DH / 32;  // fold warps (they hold the O^T rows)
    // S^T: A = K tile, B = Q (bf16, K-major).  O^T: A = V tile read MN-major,
    // B = P^T MN-major (fp16).
    constexpr uint32_t IDESC_S = idesc_bf16(128, NQ);
    constexpr uint32_t IDESC_O = idesc_f16_mn(128, NQ);
    extern __shared__ unsigned char smem_raw[];
    unsigned char* sm = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    float* red = (float*)(sm + S::OFF_RED);      // [2][4][32] reduction scratch
    float* seg_ref = red + 256;                  // [2][32] reference of the segment in each O^T buffer
    float* or_ref = red + 320;                   // [32] reference of the running output
    float* fin = red + 352;                      // [2][32] final reference and sum
    int* tinfo = (int*)(red + 416);              // [NSTG] tile's segment << 1 | accumulate
    uint64_t* bars = (uint64_t*)(sm + S::OFF_BAR);
    uint64_t* qfull = bars;
    uint64_t* kfull = bars + 1;
    uint64_t* vfull = kfull + NSTG;
    uint64_t* pready = vfull + NSTG;
    uint64_t* stfree = pready + NSTG;
    uint64_t* sfull = stfree + NSTG;
    uint64_t* ofull = sfull + 2;   // a segment's accumulation in buffer j is complete
    uint64_t* oempty = ofull + 2;  // buffer j has been folded
    uint32_t* tslot = (uint32_t*)(sm + S::OFF_MISC);
    int* flag = (int*)(sm + S::OFF_MISC + 4);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    // barriers before the dependency wait (no global memory involved)
    if (tid == 0) {
        mbar_init(qfull, 1);
        for (int j = 0; j < NSTG; ++j) {
            mbar_init(&kfull[j], 1);
            mbar_init(&vfull[j], 1);
            mbar_init(&pready[j], 4);
            mbar_init(&stfree[j], 1);
        }
        for (int j = 0; j < 2; ++j) {
            mbar_init(&sfull[j], 1);
            mbar_init(&ofull[j], 1);
            mbar_init(&oempty[j], NMW);
        }
        mbar_fence_init();
        *flag = 0;
    }
    pdl_wait();
    // ---- the item: (query block, head, sequence) and this CTA's key split
    const int h = blockIdx.y;
    const int zs = blockIdx.z / a.nsplit, split = blockIdx.z % a.nsplit;
    const int seq = a.g0 / a.q_per_seq + zs;
    const int r_lo = max(0, seq * a.q_per_seq - a.g0);
    const int r_hi = min(a.count, (seq + 1) * a.q_per_seq - a.g0);
    const int rb = r_lo + blockIdx.x * QV;
    const int re = min(rb + QV, r_hi);
    if (rb >= re) return;
    const int s = a.row_seq[rb];
    if (s < 0) return;  // rows of one sequence are all active or all inactive
    const int nq = re - rb;
    // the rows of a sequence hold consecutive positions: query q sits at
    // position pos0 + q and sees keys 0 .. pos0 + q
    const int pos0 = a.row_pos[rb];
    const int nkeys = pos0 + nq;
    const int per = ((nkeys + a.nsplit - 1) / a.nsplit + 127) & ~127;
    const int k0 = split * per, k1 = min(nkeys, k0 + per);
    if (k0 >= k1) return;
    const int nonempty = (nkeys + per - 1) / per;
    const int ntiles = (k1 - k0 + 127) >> 7;
    const int row0 = ((a.layer * a.Bmax + s) * a.nh + h) * a.n_max;  // first row of the item in the K / V maps

    __syncwarp();
    if (warp == 0) tmem_alloc(tslot, S::TCOLS);
    if (tid == 0) {
        // self-check of the operand layout: tile bases on the 1 KB swizzle
        // repeat, everything inside the dynamic shared memory (including the
        // shifted rows the V^T operand reads past its tile), TMA inner
        // coordinate on a 16-byte boundary, consecutive row positions; a
        // failure is recorded in *a.err and the CTA issues nothing
        const uint32_t end = smem_u32(smem_raw) + S::SMEM;
        int code = 0;
        if ((smem_u32(sm) & 1023) != 0) code = 41;
        else if (smem_u32(sm) + S::OFF_MISC + 8 > end || smem_u32(sm) + S::TILE + 1024 * (128 / DH) > end) code = 42;
        else if (((h * DH * 2) & 15) != 0 || a.row_pos[re - 1] != pos0 + nq - 1) code = 43;
        if (code && a.err) atomicCAS(a.err, 0, code);
        *flag = code;
    }
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    if (*flag) {
        if (warp == 0) tmem_dealloc(tmem, S::TCOLS);
        return;
    }
    const uint32_t sbase = smem_u32(sm);

    if (warp == 4) {
        // ================= producer: TMA copies and MMAs (one thread)
        if (lane == 0) {
            bool ok = true;
            int issued = 0;   // tiles whose copies are issued
            int o_done = 0;   // tiles whose O^T MMAs are issued
            int cur_seg = -1; // segment of the last O^T issued
            auto issue = [&](int t) {
                const int st = t % NSTG;
                unsigned char* stg = sm + st * S::STAGE;
                const int row = row0 + k0 + 128 * t;
                mbar_arrive_expect_tx(&kfull[st], S::TILE);
                tma_load_2d(stg + S::K_OFF, &mapK, &kfull[st], 0, row);
                mbar_arrive_expect_tx(&vfull[st], S::TILE);
                tma_load_2d(stg + S::V_OFF, &mapV, &vfull[st], 0, row);
                issued = t + 1;
            };
            mbar_arrive_expect_tx(qfull, NQ * ROWB);
            tma_load_2d(sm + S::OFF_Q, &mapQ, qfull, h * DH, rb);
            for (int t = 0; t < NSTG && t < ntiles; ++t) issue(t);
            auto do_o = [&](int u) -> bool {
                const int su = u % NSTG;
                const uint32_t pu = (uint32_t)((u / NSTG) & 1);
                if (!mbar_wait(&pready[su], pu, a.err, 51)) return false;
                const int info = tinfo[su];
                const int seg = info >> 1, ob = seg & 1;
                const bool acc = (info & 1) != 0;
                if (!acc) {
                    // a new segment: the previous one is complete, and this
                    // buffer's segment before last must have been folded
                    if (cur_seg >= 0) tc_commit(&ofull[cur_seg & 1]);
                    if (seg >= 2 && !mbar_wait(&oempty[ob], (uint32_t)(((seg - 2) >> 1) & 1), a.err, 53)) return false;
                    cur_seg = seg;
                }
                if (!mbar_wait(&vfull[su], pu, a.err, 52)) return false;
                tc_fence_after();
                const uint32_t stg = sbase + su * S::STAGE;
                const uint32_t vt = stg + S::V_OFF, pt = stg + S::K_OFF;
                const uint32_t dO = tmem + (uint32_t)(2 * NQ + ob * NQ);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {
                    // A = V^T: M = 128 spans 128 / DH swizzle-atom columns; the
                    // ones past the first read rows 1 KB further on (inside the
                    // stage), giving rows >= DH of O^T that are never read
                    tc_mma_bf16(dO, smem_desc(vt + ks * 2 * SBO_KV, 1024, SBO_KV, LAY_KV),
                                smem_desc(pt + ks * 2 * SBO_P, 16, SBO_P, LAY_P), IDESC_O, acc || ks != 0);
                }
                tc_commit(&stfree[su]);
                o_done = u + 1;
                // refill the stage with tile u + NSTG once the MMA that reads it completes
                if (u + NSTG < ntiles) {
                    if (!mbar_wait(&stfree[su], pu, a.err, 54)) return false;
                    issue(u + NSTG);
                }
                return true;
            };
            for (int t = 0; t < ntiles && ok; ++t) {
                const int st = t % NSTG, sb = t & 1;
                const uint32_t ph = (uint32_t)((t / NSTG) & 1);
                ok = (t > 0 || mbar_wait(qfull, 0, a.err, 55)) && mbar_wait(&kfull[st], ph, a.err, 56);
                if (!ok) break;
                tc_fence_after();
                // S^T of tile t into TMEM buffer t % 2 (read by the softmax of
                // tile t - 2 before its pready, which the O^T MMA of tile t - 2,
                // issued earlier by this thread, waited for)
#pragma unroll
                for (int ks = 0; ks < DH / 16; ++ks)
                    tc_mma_bf16(tmem + (uint32_t)(sb * NQ), smem_desc(sbase + st * S::STAGE + S::K_OFF + ks * 32, 16, SBO_KV, LAY_KV),
                                smem_desc(sbase + S::OFF_Q + ks * 32, 16, SBO_KV, LAY_KV), IDESC_S, ks > 0);
                tc_commit(&sfull[sb]);
                if (t >= 1) ok = do_o(t - 1);
            }
            if (ok) ok = do_o(ntiles - 1);
            if (ok && cur_seg >= 0) tc_commit(&ofull[cur_seg & 1]);  // the last segment is complete
            if (!ok) {
                // a bounded wait ran out: record it, then let this CTA's
                // copies and MMAs drain (bounded again) before returning
                atomicExch(flag, 1);
                for (int u = 0; u < issued; ++u) {
                    mbar_wait(&kfull[u % NSTG], (uint32_t)((u / NSTG) & 1), nullptr, 0);
                    mbar_wait(&vfull[u % NSTG], (uint32_t)((u / NSTG) & 1), nullptr, 0);
                }
                mbar_wait(qfull, 0, nullptr, 0);
                for (int u = 0; u < o_done; ++u) mbar_wait(&stfree[u % NSTG], (uint32_t)((u / NSTG) & 1), nullptr, 0);
            }
        }
    } else {
        // ================= softmax warps 0-3 (thread = key of the tile)
        float mref[QV], lsum[QV];  // per-query reference (base 2) and this thread's partial sum
        float Or[QV];              // threads t < DH: running output row dh = t (reference or_ref)
#pragma unroll
        for (int q = 0; q < QV; ++q) { mref[q] = -INFINITY; lsum[q] = 0.f; Or[q] = 0.f; }
        if (tid < 32) or_ref[tid] = -INFINITY;
        int seg = -1;
        const uint32_t tq = tmem + ((uint32_t)(warp * 32) << 16);
        bool ok = true;
        // fold the finished accumulation of segment sg into the running output
        auto fold = [&](int sg) -> bool {
            const int ob = sg & 1;
            bool okw = mbar_wait(&ofull[ob], (uint32_t)((sg >> 1) & 1), a.err, 57);
            okw = __all_sync(0xffffffffu, okw);
            if (okw) {
                tc_fence_after();
                float oc[LC];
                tmem_ld_cols<LC>(tq + (uint32_t)(2 * NQ + ob * NQ), oc);
#pragma unroll
                for (int q = 0; q < QV; ++q) {
                    const float ro = or_ref[q], rs = seg_ref[ob * 32 + q];
                    const float fa = ro == -INFINITY ? 0.f : exp2f(ro - rs);  // rs >= ro
                    Or[q] = Or[q] * fa + oc[q];
                }
                tc_fence_before();
            }
            __syncwarp();
            if constexpr (NMW > 1) named_sync(2, 32 * NMW);  // every fold warp has read or_ref
            if (okw && warp == 0) or_ref[lane] = seg_ref[ob * 32 + lane];
            if (okw && lane == 0) mbar_arrive(&oempty[ob]);
            __syncwarp();
            if constexpr (NMW > 1) named_sync(2, 32 * NMW);
            return okw;
        };
        for (int t = 0; t < ntiles; ++t) {
            const int st = t % NSTG, sb = t & 1;
            const uint32_t ph = (uint32_t)((t / NSTG) & 1);
            const int kt0 = k0 + 128 * t;
            const int valid = min(128, k1 - kt0);
            bool okw = mbar_wait(&sfull[sb], (uint32_t)((t >> 1) & 1), a.err, 58);
            okw = __all_sync(0xffffffffu, okw);
            if (!okw) atomicExch(flag, 1);
            tc_fence_after();
            const int qlo = max(0, kt0 + tid - pos0);  // first query that sees this key
            const bool kin = tid < valid;
            float x[QV];  // scaled scores, -inf where masked
            {
                float sc[LC];
                if (okw) tmem_ld_cols<LC>(tq + (uint32_t)(sb * NQ), sc);
#pragma unroll
                for (int q = 0; q < QV; ++q) x[q] = (okw && kin && q >= qlo && q < nq) ? sc[q] * a.c2 : -INFINITY;
            }
            bool need = t == 0;
#pragma unroll
            for (int q = 0; q < QV; ++q) need = need || x[q] > mref[q] + a.slack;
            __syncwarp();
            need = named_sync_or(1, 128, need);
            ok = named_sync_and(1, 128, okw && *flag == 0);
            if (!ok) break;
            bool acc = true;
            if (need) {
                // a new reference: the tile's per-query maximum over the four warps
                warp_red_write<QV, true>(x, red, warp, lane);
                __syncwarp();
                named_sync(1, 128);
#pragma unroll
                for (int q = 0; q < QV; ++q) {
                    const float mn = fmaxf(mref[q], warp_red_read<true>(red, q));
                    lsum[q] *= mref[q] == -INFINITY ? 0.f : exp2f(mref[q] - mn);
                    mref[q] = mn;
                }
                ++seg;
                acc = false;
                if (warp == 0) {
                    float r = -INFINITY;
#pragma unroll
                    for (int q = 0; q < QV; ++q)
                        if (q == lane) r = mref[q];
                    seg_ref[(seg & 1) * 32 + lane] = r;
                }
                __syncwarp();
                named_sync(1, 128);  // red is rewritten by a later reduction
            }
            // ---- P = fp16(2^(s - m)), partial sums, P^T over the consumed K tile
            {
                uint32_t hw[NQ / 2];
#pragma unroll
                for (int i = 0; i < NQ / 2; ++i) {
                    const int q0 = 2 * i, q1 = 2 * i + 1;
                    float p0 = 0.f, p1 = 0.f;
                    if (q0 < QV) p0 = x[q0] == -INFINITY ? 0.f : exp2f(x[q0] - mref[q0]);
                    if (q1 < QV) p1 = x[q1] == -INFINITY ? 0.f : exp2f(x[q1] - mref[q1]);
                    const __half2 pb = __floats2half2_rn(p0, p1);
                    hw[i] = *reinterpret_cast<const uint32_t*>(&pb);
                    const float2 pr = __half22float2(pb);  // the sums add the rounded weights
                    if (q0 < QV) lsum[q0] += pr.x;
                    if (q1 < QV) lsum[q1] += pr.y;
                }
                unsigned char* pP = sm + st * S::STAGE + S::K_OFF;
#pragma unroll
                for (int c = 0; c < S::PROW / 16; ++c)
                    *reinterpret_cast<uint4*>(pP + swz64_off(tid, c)) = make_uint4(hw[4 * c], hw[4 * c + 1], hw[4 * c + 2], hw[4 * c + 3]);
            }
            if (tid == 0) tinfo[st] = (seg << 1) | (acc ? 1 : 0);
            // V rows past the tile's keys (cache positions this pass never
            // wrote, possibly any bit pattern) -> 0, so that P = 0 there gives 0
            if (valid < 128) {
                bool okv = mbar_wait(&vfull[st], ph, a.err, 59);
                okv = __all_sync(0xffffffffu, okv);
                if (okv && tid >= valid) {
                    unsigned char* row = sm + st * S::STAGE + S::V_OFF + tid * ROWB;
#pragma unroll
                    for (int c = 0; c < ROWB / 16; ++c) *reinterpret_cast<uint4*>(row + 16 * c) = make_uint4(0, 0, 0, 0);
                }
                if (!okv) atomicExch(flag, 1);
            }
            fence_proxy_async_smem();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&pready[st]);
            // a segment ended: fold it (its last O^T MMA was issued or will be soon)
            if (!acc && seg >= 1 && warp < NMW) {
                if (!fold(seg - 1)) atomicExch(flag, 1);
            }
        }
        // the sums over the four warps, then the last segment's fold (the
        // decision reduced over the barrier, so the fold warps agree)
        warp_red_write<QV, false>(lsum, red, warp, lane);
        __syncwarp();
        ok = named_sync_and(1, 128, ok && *flag == 0 && seg >= 0);
        if (ok && warp < NMW) {
            if (!fold(seg)) atomicExch(flag, 1);
        }
        if (warp == 0) {  // final reference and sum per query
            float r = -INFINITY;
#pragma unroll
            for (int q = 0; q < QV; ++q)
                if (q == lane) r = mref[q];
            fin[lane] = r;
            fin[32 + lane] = warp_red_read<false>(red, lane);
        }
        __syncwarp();
        __syncthreads();
        tc_fence_after();
        if (warp == 0) tmem_dealloc(tmem, S::TCOLS);
        if (*flag) return;
        auto finish = [&](int q, float O, float L, float M) {
            const size_t row = (size_t)(rb + q);
            if (a.attnhp) {  // a = sum f v / (1 + sum f) with f = 2^(s c); h <- h + tanh(a)
                const size_t xi = row * a.d + h * DH + tid;
                const float hn = a.x[xi] + tanhf(O / (L + exp2f(-M)));
                a.x[xi] = hn;
                a.hb[row * 2 * a.d + a.d + h * DH + tid] = __float2bfloat16_rn(hn);
            } else {
                a.out[row * a.d + h * DH + tid] = __float2bfloat16_rn(O / L);
            }
        };
        if (nonempty == 1) {
            if (tid < DH) {
#pragma unroll
                for (int q = 0; q < QV; ++q)
                    if (q < nq) finish(q, Or[q], fin[32 + q], fin[q]);
            }
            pdl_trigger();
            return;
        }
        // ---- split: publish the partial, the last CTA of the item merges
        const int item = (zs * gridDim.y + h) * gridDim.x + blockIdx.x;
        const size_t slot = (size_t)item * a.nsplit + split;
        float* po = a.part + slot * (size_t)(NQ * (DH + 2));
        if (tid < DH) {
#pragma unroll
            for (int q = 0; q < QV; ++q) po[q * DH + tid] = Or[q];
        }
        if (tid < QV) {
            po[NQ * DH + 2 * tid] = fin[tid];
            po[NQ * DH + 2 * tid + 1] = fin[32 + tid];
        }
        __threadfence();
        __syncwarp();
        named_sync(1, 128);
        if (tid == 0) *flag = atomicAdd(&a.cnt[item], 1) == nonempty - 1 ? 2 : 0;
        __syncwarp();
        named_sync(1, 128);
        if (*flag != 2) {
            pdl_trigger();
            return;
        }
        __threadfence();
        if (tid < DH) {
            const float* base = a.part + (size_t)item * a.nsplit * (NQ * (DH + 2));
            for (int q = 0; q < nq && q < QV; ++q) {
                float M = -INFINITY;
                for (int sp = 0; sp < nonempty; ++sp) M = fmaxf(M, base[(size_t)sp * NQ * (DH + 2) + NQ * DH + 2 * q]);
                float O = 0.f, L = 0.f;
                for (int sp = 0; sp < nonempty; ++sp) {
                    const float* b = base + (size_t)sp * NQ * (DH + 2);
                    const float ms = b[NQ * DH + 2 * q];
                    if (ms == -INFINITY) continue;
                    const float e = exp2f(ms - M);
                    O += b[q * DH + tid] * e;
                    L += b[NQ * DH + 2 * q + 1] * e;
                }
                finish(q, O, L, M);
            }
        }
        if (tid == 0) a.cnt[item] = 0;  // ready for the next launch
        pdl_trigger();
        return;
    }
    // producer warp: join the CTA barrier, then leave
    __syncwarp();
    __syncthreads();
    pdl_trigger();
}

// ---------------------------------------------------------------- host side
static CUtensorMapSwizzle swz_enum(int rowb) {
    return rowb == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : rowb == 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B;
}

// KV cache [items * n_max rows][dh] as a 2-D map, boxes of box_rows rows,
// swizzled by the row width (32, 64 or 128 bytes).
bool kv_tile_map(CUtensorMap* m, const void* base, int dh, int n_max, long long items, int box_rows, int f16) {
    auto enc = tmap_encoder();
    if (!enc || ((uintptr_t)base & 15) || items * n_max >= (1LL << 31)) return false;
    if (!(dh == 16 || dh == 32 || dh == 64) || box_rows < 1 || box_rows > 256) return false;
    cuuint64_t dims[2] = {(cuuint64_t)dh, (cuuint64_t)(items * n_max)};
    cuuint64_t strides[1] = {(cuuint64_t)dh * 2};
    cuuint32_t box[2] = {(cuuint32_t)dh, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base),
               dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz_enum(dh * 2),
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Q rows [R][d] as a 2-D map, boxes of nq rows x dh columns.
static bool q_map(CUtensorMap* m, const void* base, int d, int R, int dh, int nq) {
    auto enc = tmap_encoder();
    if (!enc || ((uintptr_t)base & 15)) return false;
    cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)R};
    cuuint64_t strides[1] = {(cuuint64_t)d * 2};
    cuuint32_t box[2] = {(cuuint32_t)dh, (cuuint32_t)nq};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, swz_enum(dh * 2), CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DH, int QV>
static cudaError_t launch_tc_t(const CUtensorMap& mk, const CUtensorMap& mv, const CUtensorMap& mq,
                               const AttTcArgs& a, dim3 grid, cudaStream_t st) {
    const int sm = AttTcShape<DH>::SMEM;
    cudaError_t e = cudaFuncSetAttribute(k_attn_tc<DH, QV>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
    if (e != cudaSuccess) return e;
    return launch_k(k_attn_tc<DH, QV>, grid, dim3(160), (size_t)sm, st, mk, mv, mq, a);
}

// Tiles one CTA walks at most before the key range is split across CTAs.
constexpr int ATT_MAX_TILES = 8;

int attn_tc_supported(int dh) { return dh == 32 || dh == 64; }

long long attn_splits(long long items, int n_max, int dh, int nq, int n_sm) {
    (void)dh; (void)nq;
    // enough CTAs to cover the GPU about twice over (four CTAs per SM), and
    // no CTA walking more than ATT_MAX_TILES tiles of 128 keys
    const long long want = (2LL * 4 * n_sm + items - 1) / items;
    const long long by_len = (n_max + 128LL * ATT_MAX_TILES - 1) / (128LL * ATT_MAX_TILES);
    long long ns = want > by_len ? want : by_len;
    const long long max_ns = (n_max + 127) / 128;
    if (ns > max_ns) ns = max_ns;
    if (ns > 64) ns = 64;
    return ns < 1 ? 1 : ns;
}

cudaError_t launch_attn_tc(const AttArgs<bf16>& aa, int dh, int nh, int nseg, bool step_rows,
                           const AttnScratch& sc, int* err, cudaStream_t st) {
    static int n_sm = 0;
    if (!n_sm) {
        int dev = 0;
        cudaGetDevice(&dev);
        if (cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n_sm <= 0) n_sm = 148;
    }
    constexpr int NQ = 32;
    const int QV = aa.q_per_seq == 1 ? 1 : aa.q_per_seq <= 16 ? 16 : 32;  // query rows per CTA
    const int qblocks = (aa.q_per_seq + QV - 1) / QV;
    const long long items = (long long)qblocks * nh * nseg;
    const long long kv_items = (long long)(aa.layer + 1) * aa.kv.Bmax * nh;  // items up to this layer
    CUtensorMap mk, mv, mq;
    if (!kv_tile_map(&mk, aa.kc, dh, aa.kv.n_max, kv_items, 128) || !kv_tile_map(&mv, aa.vc, dh, aa.kv.n_max, kv_items, 128, 1) ||
        !q_map(&mq, aa.q, aa.d, aa.count, dh, NQ))
        return cudaErrorInvalidValue;
    AttTcArgs a{};
    a.row_seq = aa.row_seq; a.row_pos = aa.row_pos;
    a.out = aa.out; a.x = aa.x; a.hb = aa.hb;
    a.count = aa.count; a.q_per_seq = aa.q_per_seq; a.g0 = aa.g0; a.d = aa.d; a.nh = nh;
    a.layer = aa.layer; a.Bmax = aa.kv.Bmax; a.n_max = aa.kv.n_max; a.attnhp = aa.attnhp;
    a.c2 = aa.scale * 1.4426950408889634f;
    // reference slack of the softmax (below 16 keeps P inside fp16);
    // TPPSD_ATTN_SLACK lowers it to exercise the reference changes in tests
    const char* slack = getenv("TPPSD_ATTN_SLACK");
    a.slack = slack ? (float)atof(slack) : 15.f;
    a.err = err;
    // key splits: only for one-pass (step) rows
    int nsplit = 1;
    if (step_rows && sc.part && sc.cnt) {
        long long ns = attn_splits(items, aa.kv.n_max, dh, NQ, n_sm);
        if (const char* f = getenv("TPPSD_ATTN_SPLITS")) ns = atoi(f) > 0 ? atoi(f) : ns;
        const size_t slot_bytes = (size_t)NQ * (dh + 2) * 4;
        while (ns > 1 && ((size_t)(items * ns) * slot_bytes > sc.part_bytes || items > sc.cnt_items)) --ns;
        nsplit = (int)ns;
    }
    if ((long long)nseg * nsplit > 65535) return cudaErrorInvalidValue;
    a.nsplit = nsplit;
    a.part = sc.part;
    a.cnt = sc.cnt;
    const dim3 grid(qblocks, nh, nseg * nsplit);
    cudaError_t e;
#define ATT_TC_QV(DH)                                                  \
    (QV == 1 ? launch_tc_t<DH, 1>(mk, mv, mq, a, grid, st)                \
             : QV == 16 ? launch_tc_t<DH, 16>(mk, mv, mq, a, grid, st)     \
                        : launch_tc_t<DH, 32>(mk, mv, mq, a, grid, st))
    switch (dh) {
        case 32: e = ATT_TC_QV(32); break;
        case 64: e = ATT_TC_QV(64); break;
        default: return cudaErrorInvalidValue;
    }
#undef ATT_TC_QV
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tppsd
