// Tensor-core GEMM for the target model's linear layers (bf16 in, fp32
// accumulate): Y[R][N] = A[R][K] W[N][K]^T + b, with the epilogue fused.
//
// One CTA computes a 128 x BN tile.  Warp 0 (one thread) streams 128x64 A
// and BNx64 W tiles into shared memory with TMA (128-byte swizzle) through
// a ring of stages guarded by mbarriers; warp 1 (one thread) issues
// tcgen05.mma (M=128, N<=256 per instruction, K=16) into a TMEM
// accumulator and releases each stage with tcgen05.commit; then all four
// warps read the accumulator back (thread t owns row t of the tile: TMEM
// lane t) and apply the epilogue; warps 2-3, idle during the main loop,
// stage the epilogue's parameters in shared memory meanwhile:
//   EPI_QKV      bias, bf16 round, Q to the row buffer, K/V scattered into the
//                KV cache at each row's (sequence, position)
//   EPI_RELU     bias, ReLU, bf16 round
//   EPI_F32      bias, fp32 rows (the heads' [E; V_k1] h)
// In the split form an fp32-accurate product of fp32 operands, each given
// as two bf16 parts (x = x_hi + x_lo), runs as one GEMM over three times the
// K blocks: A_hi W_hi + A_hi W_lo + A_lo W_hi (the K loop walks the three
// pairs of maps; the dropped A_lo W_lo term is below 2^-16 of |A| |W|).
// The residual + LayerNorm epilogue (rows of N = d) is k_gemm_ln_cl below.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cuda_fp16.h>

#include "common.cuh"
#include "engine.h"
#include "tc_ptx.cuh"

namespace tppsd {

template <int BN>
struct TcShape {
    static constexpr int BM = 128, BK = 64;
    static constexpr int STAGES = BN >= 512 ? 2 : 4;
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int STAGE = A_BYTES + B_BYTES;
    static constexpr int TMEM_COLS = BN < 32 ? 32 : BN;
    // epilogue parameters staged in shared memory: bias[BN], row seq/pos[BM]
    static constexpr int PARAM_BYTES = BN * 4 + 2 * BM * 4;
    static constexpr size_t SMEM = (size_t)STAGES * STAGE + PARAM_BYTES + 1024 + 256;
};


template <int BN>
__global__ void __launch_bounds__(128, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
              const __grid_constant__ CUtensorMap mapA2, const __grid_constant__ CUtensorMap mapB2, TcGemmArgs a) {
    using S = TcShape<BN>;
    // Before griddepcontrol.wait nothing reads what the previous kernel of
    // the stream writes: barrier set-up, TMEM allocation and the weight
    // tiles of the first stages (the weights are never written by a
    // sampling kernel) overlap that kernel's tail; every role waits before
    // its first dependent access (rows, row positions, outputs).
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    float* bias_s = (float*)(smem + S::STAGES * S::STAGE);
    int* rseq_s = (int*)(bias_s + BN);
    int* rpos_s = rseq_s + S::BM;
    uint64_t* full = (uint64_t*)(rpos_s + S::BM);
    uint64_t* empty = full + S::STAGES;
    uint64_t* done = empty + S::STAGES;
    uint32_t* tslot = (uint32_t*)(done + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n0 = blockIdx.x * BN, m0 = blockIdx.y * S::BM;
    const int KB = a.K / S::BK, KBT = a.split ? 3 * KB : KB;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(done, 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(tslot, S::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;

    if (a.stall) {
        // Diagnostic requested by the host: wait on the completion barrier
        // before anything is issued.  Nothing can complete it, so the bounded
        // wait runs out, records its code in *a.err and the CTA returns with
        // no copy or MMA in flight.
        pdl_wait();
        if (threadIdx.x == 0) mbar_wait(done, 0, a.err, 9);
        __syncthreads();
        if (warp == 0) tmem_dealloc(tmem, S::TMEM_COLS);
        return;
    }

    if (warp == 0 && lane == 0) {
        // producer: TMA loads of the A and W tiles of every K block; the W
        // tiles of the first stages go out before the wait
        const int pre = KBT < S::STAGES ? KBT : S::STAGES;
        auto load_w = [&](int kb, int s) {
            const int pair = kb / KB, kx = (kb - pair * KB) * S::BK;  // split: (hi, hi), (hi, lo), (lo, hi)
#pragma unroll
            for (int c = 0; c < BN; c += 256)
                tma_load_2d(smem + s * S::STAGE + S::A_BYTES + c * 128, pair == 1 ? &mapB2 : &mapB, &full[s], kx,
                            n0 + c);
        };
        for (int kb = 0; kb < pre; ++kb) {
            mbar_arrive_expect_tx(&full[kb], S::STAGE);
            load_w(kb, kb);
        }
        pdl_wait();
        for (int kb = 0; kb < KBT; ++kb) {
            const int s = kb % S::STAGES, round = kb / S::STAGES;
            if (kb >= pre) {
                if (!mbar_wait(&empty[s], (round & 1) ^ 1, a.err, 1)) break;
                mbar_arrive_expect_tx(&full[s], S::STAGE);
                load_w(kb, s);
            }
            const int pair = kb / KB, kx = (kb - pair * KB) * S::BK;
            tma_load_2d(smem + s * S::STAGE, pair == 2 ? &mapA2 : &mapA, &full[s], kx, m0);
        }
    } else if (warp == 1 && lane == 0) {
        // MMA issuer
        constexpr int NI = BN < 256 ? BN : 256;
        const uint32_t idesc = idesc_bf16(128, NI);
        for (int kb = 0; kb < KBT; ++kb) {
            const int s = kb % S::STAGES, round = kb / S::STAGES;
            if (!mbar_wait(&full[s], round & 1, a.err, 2)) break;
            tc_fence_after();
            const uint32_t abase = smem_u32(smem + s * S::STAGE), bbase = abase + S::A_BYTES;
#pragma unroll
            for (int kk = 0; kk < S::BK / 16; ++kk) {
                const uint64_t ad = sw128_desc(abase + kk * 32);
#pragma unroll
                for (int c = 0; c < BN; c += 256)
                    tc_mma_bf16(tmem + c, ad, sw128_desc(bbase + c * 128 + kk * 32), idesc,
                                (kb | kk) != 0);
            }
            tc_commit(&empty[s]);
        }
        tc_commit(done);  // arrives when every MMA above has completed
    } else if (warp >= 2) {
        // idle during the main loop: stage the epilogue's parameters
        const int t = threadIdx.x - 64;
        for (int c = t; c < BN; c += 64) bias_s[c] = a.bias[n0 + c];
        pdl_wait();
        if (a.epi == EPI_TC_QKV) {
            for (int r = t; r < S::BM; r += 64) {
                const bool in = m0 + r < a.R;
                rseq_s[r] = in ? a.row_seq[m0 + r] : -1;
                rpos_s[r] = in ? a.row_pos[m0 + r] : 0;
            }
        }
    }
    __syncwarp();
    if (warp < 2) pdl_wait();  // the epilogue writes what the previous kernel may read
    const bool ok = __syncthreads_and(mbar_wait(done, 0, a.err, 3)) != 0;  // CTA-uniform
    tc_fence_after();
    // the next kernel may be scheduled now: its CTAs set up (and wait for
    // this grid's completion) while the epilogues run
    pdl_trigger();

    const int t = warp * 32 + lane, r = m0 + t;
    const bool live = ok && r < a.R;
    const uint32_t tw = tmem + ((uint32_t)(warp * 32) << 16);
    if (ok) {
        if (a.epi == EPI_TC_F32) {
            for (int c0 = 0; c0 < BN; c0 += 16) {
                float v[16];
                tmem_ld16(tw + c0, v);
                if (live) {
                    float4* o = reinterpret_cast<float4*>(a.out_f + (size_t)r * a.N + n0 + c0);
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        o[i] = make_float4(v[4 * i] + bias_s[c0 + 4 * i], v[4 * i + 1] + bias_s[c0 + 4 * i + 1],
                                           v[4 * i + 2] + bias_s[c0 + 4 * i + 2], v[4 * i + 3] + bias_s[c0 + 4 * i + 3]);
                }
            }
        } else if (a.epi == EPI_TC_RELU) {
            for (int c0 = 0; c0 < BN; c0 += 16) {
                float v[16];
                tmem_ld16(tw + c0, v);
                if (live) {
#pragma unroll
                    for (int i = 0; i < 16; ++i) v[i] = fmaxf(v[i] + bias_s[c0 + i], 0.f);
                    st_bf16x16(a.out_t + (size_t)r * a.N + n0 + c0, v);
                }
            }
        } else {  // EPI_TC_QKV
            const int s = live ? rseq_s[t] : -1, pos = rpos_s[t];
            for (int c0 = 0; c0 < BN; c0 += 16) {
                float v[16];
                tmem_ld16(tw + c0, v);
                if (!live) continue;
                const int col = n0 + c0, which = col / a.d, cc = col - which * a.d;
#pragma unroll
                for (int i = 0; i < 16; ++i) v[i] += bias_s[c0 + i];
                if (which == 0) {
                    st_bf16x16(a.q_out + (size_t)r * a.d + cc, v);
                } else if (s >= 0) {
                    const int h = cc / a.dh, e = cc - h * a.dh;
                    const size_t o = ((((size_t)a.layer * a.Bmax + s) * a.nh + h) * (size_t)a.n_max + pos) * a.dh + e;
                    if (which == 2 && a.v_f16) st_f16x16_of_bf16(a.vc + o, v);
                    else st_bf16x16((which == 1 ? a.kc : a.vc) + o, v);
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, S::TMEM_COLS);
    pdl_trigger();
}

// ---------------------------------------------------------------- LayerNorm GEMM
// Y = LayerNorm(A W^T + b + resid) over rows of N = CL * BNC columns.  A
// cluster of CL CTAs shares 128 rows, CTA j computing columns j*BNC ..
// (j+1)*BNC - 1 on the tensor cores, so a row's LayerNorm statistics are
// summed over the cluster through distributed shared memory (two-pass:
// mean, then the centred sum of squares).  Thread t owns row t of the tile.
// The residual rows of the CTA's columns are prefetched by bulk copies
// while the main loop runs.
template <int BNC>
struct LnShape {
    static constexpr int BM = 128, BK = 64, STAGES = 4;
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = BNC * BK * 2;
    static constexpr int STAGE = A_BYTES + B_BYTES;
    static constexpr int RLD = BNC + 4;              // padded residual row (floats)
    static constexpr int RES_BYTES = BM * RLD * 4;
    static constexpr int TMEM_COLS = BNC;
    static constexpr size_t SMEM = (size_t)STAGES * STAGE + RES_BYTES + 2 * BM * 4 + 3 * BNC * 4 + 1024 + 256;
};

template <int BNC>
__global__ void __launch_bounds__(128, 1)
    k_gemm_ln_cl(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB, TcGemmArgs a) {
    using S = LnShape<BNC>;
    extern __shared__ unsigned char smem_raw[];
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    float* resid_s = (float*)(smem + S::STAGES * S::STAGE);
    float* red1 = resid_s + S::BM * S::RLD;
    float* red2 = red1 + S::BM;
    float* prm = red2 + S::BM;  // bias, LN gain, LN shift of the CTA's columns
    uint64_t* full = (uint64_t*)(prm + 3 * BNC);
    uint64_t* empty = full + S::STAGES;
    uint64_t* done = empty + S::STAGES;
    uint64_t* resbar = done + 1;
    uint32_t* tslot = (uint32_t*)(resbar + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t crank = cluster_ctarank(), ncl = cluster_nctarank();
    const int n0 = (int)crank * BNC, m0 = blockIdx.y * S::BM;
    const int KB = a.K / S::BK, N = a.N;
    const int rows = min(S::BM, a.R - m0);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(done, 1);
        mbar_init(resbar, 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(tslot, S::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;

    if (warp == 0 && lane == 0) {
        // residual rows (BNC contiguous floats each), then the A / W tiles
        mbar_arrive_expect_tx(resbar, (uint32_t)rows * BNC * 4);
        for (int r = 0; r < rows; ++r)
            bulk_load(resid_s + r * S::RLD, a.resid + (size_t)(m0 + r) * N + n0, BNC * 4, resbar);
        for (int kb = 0; kb < KB; ++kb) {
            const int s = kb % S::STAGES, round = kb / S::STAGES;
            if (!mbar_wait(&empty[s], (round & 1) ^ 1, a.err, 1)) break;
            mbar_arrive_expect_tx(&full[s], S::STAGE);
            unsigned char* st = smem + s * S::STAGE;
            tma_load_2d(st, &mapA, &full[s], kb * S::BK, m0);
            tma_load_2d(st + S::A_BYTES, &mapB, &full[s], kb * S::BK, n0);
        }
    } else if (warp == 1 && lane == 0) {
        const uint32_t idesc = idesc_bf16(128, BNC);
        for (int kb = 0; kb < KB; ++kb) {
            const int s = kb % S::STAGES, round = kb / S::STAGES;
            if (!mbar_wait(&full[s], round & 1, a.err, 2)) break;
            tc_fence_after();
            const uint32_t abase = smem_u32(smem + s * S::STAGE), bbase = abase + S::A_BYTES;
#pragma unroll
            for (int kk = 0; kk < S::BK / 16; ++kk)
                tc_mma_bf16(tmem, sw128_desc(abase + kk * 32), sw128_desc(bbase + kk * 32), idesc,
                            (kb | kk) != 0);
            tc_commit(&empty[s]);
        }
        tc_commit(done);
    } else if (warp >= 2) {
        for (int c = threadIdx.x - 64; c < BNC; c += 64) {
            prm[c] = a.bias[n0 + c];
            prm[BNC + c] = a.ln_g[n0 + c];
            prm[2 * BNC + c] = a.ln_b[n0 + c];
        }
    }
    __syncwarp();
    const bool ok = __syncthreads_and(mbar_wait(done, 0, a.err, 3)) != 0;  // CTA-uniform
    tc_fence_after();
    const bool have_res = mbar_wait(resbar, 0, a.err, 4);

    const int t = warp * 32 + lane, r = m0 + t;
    const bool live = ok && t < rows;
    const uint32_t tw = tmem + ((uint32_t)(warp * 32) << 16);
    float y[BNC];
#pragma unroll
    for (int c0 = 0; c0 < BNC; c0 += 16) {
        float v[16];
        tmem_ld16(tw + c0, v);
#pragma unroll
        for (int i = 0; i < 16; ++i) y[c0 + i] = v[i] + prm[c0 + i];
    }
    float s1 = 0.f;
    if (live) {
#pragma unroll
        for (int c = 0; c < BNC; c += 4) {
            const float4 q = have_res ? *reinterpret_cast<const float4*>(resid_s + t * S::RLD + c)
                                      : *reinterpret_cast<const float4*>(a.resid + (size_t)r * N + n0 + c);
            y[c] += q.x; y[c + 1] += q.y; y[c + 2] += q.z; y[c + 3] += q.w;
        }
#pragma unroll
        for (int c = 0; c < BNC; ++c) s1 += y[c];
    }
    red1[t] = s1;
    cluster_sync();
    float tot1 = 0.f;
    for (uint32_t j = 0; j < ncl; ++j) tot1 += ld_dsmem_f32(red1 + t, j);
    const float mean = tot1 / N;
    float s2 = 0.f;
#pragma unroll
    for (int c = 0; c < BNC; ++c) s2 += (y[c] - mean) * (y[c] - mean);
    red2[t] = s2;
    cluster_sync();
    float tot2 = 0.f;
    for (uint32_t j = 0; j < ncl; ++j) tot2 += ld_dsmem_f32(red2 + t, j);
    const float inv = 1.0f / sqrtf(tot2 / N + LN_EPS);
    if (live) {
#pragma unroll
        for (int c0 = 0; c0 < BNC; c0 += 16) {
            float o[16];
#pragma unroll
            for (int i = 0; i < 16; ++i)
                o[i] = (y[c0 + i] - mean) * inv * prm[BNC + c0 + i] + prm[2 * BNC + c0 + i];
            float4* xo = reinterpret_cast<float4*>(a.x_out + (size_t)r * N + n0 + c0);
#pragma unroll
            for (int i = 0; i < 4; ++i) xo[i] = make_float4(o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
            st_bf16x16(a.xb_out + (size_t)r * N + n0 + c0, o);
        }
    }
    cluster_sync();  // no CTA leaves while another may still read its red2
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, S::TMEM_COLS);
}

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
    }
    return fn;
}

bool make_tmap_bf16(CUtensorMap* map, const void* ptr, int K, int rows, int box_rows) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = tmap_encoder();
    if (!enc || K % 64 || ((uintptr_t)ptr & 15)) return false;
    cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)K * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN>
static cudaError_t launch_bn(const CUtensorMap& A, const CUtensorMap& W, const CUtensorMap& A2,
                             const CUtensorMap& W2, const TcGemmArgs& a, cudaStream_t st) {
    const size_t sm = TcShape<BN>::SMEM;
    cudaError_t e = cudaFuncSetAttribute(k_gemm_tc<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    const dim3 grid(a.N / BN, (a.R + 127) / 128);
    return launch_k(k_gemm_tc<BN>, grid, dim3(128), sm, st, A, W, A2, W2, a);
}

template <int BNC>
static cudaError_t launch_ln_bnc(const CUtensorMap& A, const CUtensorMap& W, const TcGemmArgs& a, int CL,
                                 cudaStream_t st) {
    const size_t sm = LnShape<BNC>::SMEM;
    cudaError_t e = cudaFuncSetAttribute(k_gemm_ln_cl<BNC>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(CL, (a.R + 127) / 128, 1);
    cfg.blockDim = dim3(128, 1, 1);
    cfg.dynamicSmemBytes = sm;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = CL;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_gemm_ln_cl<BNC>, A, W, a);
}

int ln_cluster_cols(int N) {
    if (N % 32 || N < 32) return 0;
    if (N <= 256) return 32;
    if (N <= 512 && N % 64 == 0) return 64;
    return 0;
}

cudaError_t launch_gemm_ln_cluster(const CUtensorMap& A, const CUtensorMap& W, const TcGemmArgs& a,
                                   cudaStream_t st) {
    if (a.R <= 0) return cudaSuccess;
    const int bnc = ln_cluster_cols(a.N);
    if (!bnc || a.K % 64) return cudaErrorInvalidValue;
    const int CL = a.N / bnc;
    if (CL > 8) return cudaErrorInvalidValue;
    return bnc == 32 ? launch_ln_bnc<32>(A, W, a, CL, st) : launch_ln_bnc<64>(A, W, a, CL, st);
}

cudaError_t launch_gemm_tc_split(const CUtensorMap& A, const CUtensorMap& A2, const CUtensorMap& W,
                                 const CUtensorMap& W2, const TcGemmArgs& a, int BN, cudaStream_t st) {
    if (a.R <= 0) return cudaSuccess;
    if (a.epi != EPI_TC_QKV && a.epi != EPI_TC_RELU && a.epi != EPI_TC_F32) return cudaErrorInvalidValue;
    if (a.K % 64 || a.N % BN) return cudaErrorInvalidValue;
    switch (BN) {
        case 32: return launch_bn<32>(A, W, A2, W2, a, st);
        case 64: return launch_bn<64>(A, W, A2, W2, a, st);
        case 128: return launch_bn<128>(A, W, A2, W2, a, st);
        case 256: return launch_bn<256>(A, W, A2, W2, a, st);
        case 512: return launch_bn<512>(A, W, A2, W2, a, st);
    }
    return cudaErrorInvalidValue;
}

cudaError_t launch_gemm_tc(const CUtensorMap& A, const CUtensorMap& W, const TcGemmArgs& a, int BN,
                           cudaStream_t st) {
    if (a.split) return cudaErrorInvalidValue;
    return launch_gemm_tc_split(A, A, W, W, a, BN, st);
}

}  // namespace tppsd
