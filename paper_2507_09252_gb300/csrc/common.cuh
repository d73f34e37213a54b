// Device-side building blocks shared by the kernels of the TPP-SD sampler.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace tppsd {

constexpr float LN_EPS = 1e-5f;
constexpr uint32_t FLAG_NO_BONUS = 1u;

typedef __nv_bfloat16 bf16;

// ---------------------------------------------------------------- launch order
// Programmatic dependent launch: a kernel launched with programmatic stream
// serialization may start while the previous kernel of the stream is still
// finishing; pdl_wait() blocks until that kernel has completed and its
// memory is visible, so every kernel calls it before its first access to
// global memory.  pdl_trigger() lets the next kernel start launching once
// every CTA of this one has called it or exited.  Both are no-ops for a
// kernel launched without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ---------------------------------------------------------------- storage
// Storage type T of weights, GEMM inputs and KV: float (fp32 models) or bf16.
template <typename T> struct St;
template <> struct St<float> {
    static __device__ __forceinline__ float ld(const float* p) { return *p; }
    static __device__ __forceinline__ void st(float* p, float v) { *p = v; }
    static __device__ __forceinline__ float rnd(float v) { return v; }
};
template <> struct St<bf16> {
    static __device__ __forceinline__ float ld(const bf16* p) { return __bfloat162float(*p); }
    static __device__ __forceinline__ void st(bf16* p, float v) { *p = __float2bfloat16_rn(v); }
    static __device__ __forceinline__ float rnd(float v) { return __bfloat162float(__float2bfloat16_rn(v)); }
};

// ---------------------------------------------------------------- Philox
// Philox4x32-10 as defined by Salmon et al. (SC'11): ten rounds of
// (hi, lo) = M * x on words 0 and 2, mixed with words 1, 3 and the key; the
// key is bumped by the Weyl constants between rounds.
struct U4 { float x, y, z, w; };

// Temporal encoding (App. D.4) of a model with encoding table tenc (a_j,
// then b_j; fp64) and width d: the angle a_j + b_j t formed and reduced mod
// 2 pi in fp64, then fp32 sin / cos.  Dimensions 2i, 2i+1 share one angle
// (one sincos) when paired (THP, AttNHP); SAHP's have their own.
__device__ __forceinline__ float tenc_angle(const double* tenc, int d, int j, double t) {
    const double ang = tenc[j] + tenc[d + j] * t;
    return (float)fma(-6.283185307179586476925, rint(ang * 0.15915494309189533577), ang);
}
__device__ __forceinline__ void tenc_pair_of(const double* tenc, int d, int paired, double t, int i, float* z0,
                                             float* z1) {
    float sv, cv;
    sincosf(tenc_angle(tenc, d, 2 * i, t), &sv, &cv);
    if (!paired) cv = cosf(tenc_angle(tenc, d, 2 * i + 1, t));
    *z0 = sv;
    *z1 = cv;
}

__device__ __forceinline__ uint4 philox(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t a = 0xD2511F53u * c.x, ah = __umulhi(0xD2511F53u, c.x);
        const uint32_t b = 0xCD9E8D57u * c.z, bh = __umulhi(0xCD9E8D57u, c.z);
        c = make_uint4(bh ^ c.y ^ k0, b, ah ^ c.w ^ k1, a);
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return c;
}

// Uniforms of slot (seed, seq, pos, block): counter (pos, block, seq, 0);
// word w -> ((w >> 8) + 0.5) / 2^24, exact in fp32.
__device__ __forceinline__ U4 slot_uniforms(uint64_t seed, uint32_t seq, uint32_t pos, uint32_t block) {
    uint4 r = philox(make_uint4(pos, block, seq, 0u), (uint32_t)seed, (uint32_t)(seed >> 32));
    const float s = 1.0f / 16777216.0f;
    U4 u;
    u.x = ((float)(r.x >> 8) + 0.5f) * s;
    u.y = ((float)(r.y >> 8) + 0.5f) * s;
    u.z = ((float)(r.z >> 8) + 0.5f) * s;
    u.w = ((float)(r.w >> 8) + 0.5f) * s;
    return u;
}

// ---------------------------------------------------------------- reductions
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// ---------------------------------------------------------------- head math
// Head row layout: [log w (M) | mu (M) | s = log sigma (M) | log f (K)].
// log g(tau) = logsumexp_m [log w_m - log tau - s_m - log(2 pi)/2
//                           - (log tau - mu_m)^2 / (2 exp(2 s_m))]   (Sec. 4.2)
__device__ __forceinline__ float head_log_g(const float* hd, int M, float tau) {
    const float lt = logf(tau);
    const float HALF_LOG_2PI = 0.91893853320467274178f;
    float mx = -INFINITY;
    for (int m = 0; m < M; ++m) {
        const float z = (lt - hd[M + m]) * expf(-hd[2 * M + m]);
        mx = fmaxf(mx, hd[m] - hd[2 * M + m] - 0.5f * z * z);
    }
    float acc = 0.f;
    for (int m = 0; m < M; ++m) {
        const float z = (lt - hd[M + m]) * expf(-hd[2 * M + m]);
        acc += expf(hd[m] - hd[2 * M + m] - 0.5f * z * z - mx);
    }
    return mx + logf(acc) - lt - HALF_LOG_2PI;
}

// Smallest index whose running sum of exp(logp) reaches u * total.
__device__ __forceinline__ int pick_categorical_log(const float* logp, int n, float u) {
    float tot = 0.f;
    for (int i = 0; i < n; ++i) tot += expf(logp[i]);
    const float target = u * tot;
    float run = 0.f;
    for (int i = 0; i < n; ++i) {
        run += expf(logp[i]);
        if (run >= target) return i;
    }
    return n - 1;
}

// tau = exp(mu_z + sigma_z * eps), z ~ Cat(w), eps by Box-Muller (cos branch)
// (Sec. 4.2 naive sampling, App. A.1).
__device__ __forceinline__ float draw_tau(const float* hd, int M, float u_comp, float u1, float u2) {
    const int z = pick_categorical_log(hd, M, u_comp);
    const float eps = sqrtf(-2.0f * logf(u1)) * cospif(2.0f * u2);
    return expf(hd[M + z] + expf(hd[2 * M + z]) * eps);
}

}  // namespace tppsd
