// Device helpers shared by the CyFA kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.h"

namespace cyfa {

constexpr int MS = 128;        // storage rows per state (m* = m + 1)
constexpr int MA = 127;        // active relative-time slots m
constexpr int NPAIR = 63;      // cosine-sine pairs (m - 1) / 2
constexpr float INV_SQRT_M = 0.088735650941611f;   // 1 / sqrt(127)
constexpr float SQRT_2_OVER_M = 0.125491161809579f; // sqrt(2 / 127)

__device__ __forceinline__ float ldf(const float* p, size_t i) { return p[i]; }
__device__ __forceinline__ float ldf(const __nv_bfloat16* p, size_t i) { return __bfloat162float(p[i]); }
__device__ __forceinline__ void stf(float* p, size_t i, float x) { p[i] = x; }
__device__ __forceinline__ void stf(__nv_bfloat16* p, size_t i, float x) { p[i] = __float2bfloat16_rn(x); }

// Phase of the j-th rotation block of U(lam): theta_j = 2 pi j lam / m = pi * phase_pi(lam, j).
// lam is the clock reduced mod m (in [0, m)).  lam is split as hi + lo with hi on a 1/256 grid,
// so j*hi and its reduction mod m are exact in fp32; only the small j*lo term rounds.
__device__ __forceinline__ float phase_pi(float lam, int j) {
    const float hi = rintf(lam * 256.f) * (1.f / 256.f);
    const float lo = lam - hi;
    const float jh = (float)j * hi;
    const float qn = floorf(jh * (1.f / 127.f));
    float r = fmaf(-qn, 127.f, jh);
    if (r < 0.f) r += 127.f;
    else if (r >= 127.f) r -= 127.f;
    r = fmaf((float)j, lo, r);
    return r * (2.f / 127.f);
}

// phase_pi for m active slots (the same arithmetic with m in place of 127; identical values at
// m = 127): lam in [0, m), theta_j = 2 pi j lam / m = pi * phase_pi_m(lam, j, sl).
template <class SL>
__device__ __forceinline__ float phase_pi_m(float lam, int j, const SL& sl) {
    const float hi = rintf(lam * 256.f) * (1.f / 256.f);
    const float lo = lam - hi;
    const float jh = (float)j * hi;
    const float qn = floorf(jh * sl.inv_m);
    float r = fmaf(-qn, sl.fm, jh);
    if (r < 0.f) r += sl.fm;
    else if (r >= sl.fm) r -= sl.fm;
    r = fmaf((float)j, lo, r);
    return r * sl.two_over_m;
}

// Temporal write-vector entries for one token: a = beta * U(-lam) b (Sec. 3.2), with
// b = [1/sqrt(m), sqrt(2/m), 0, sqrt(2/m), 0, ...] (App. A.1 Eq. app-b-explicit), so
// a[0] = beta/sqrt(m), a[2j-1] = beta sqrt(2/m) cos(theta_j), a[2j] = -beta sqrt(2/m) sin(theta_j)
// for j <= (m-1)/2, and the padding entries a[m..ms-1] = 0 (App. A.7).
// Fills the ms entries of rows r < C of a row-major [C][ld] shared array; row r is scaled by
// sc[r] * beta[r].
template <class ScaleFn>
__device__ __forceinline__ void build_write_rows(float* sA, int ld, const float* slam,
                                                 const float* sbeta, int C, const Slots& sl,
                                                 ScaleFn scale_of) {
    const int lg = sl.ms == 256 ? 7 : 6;   // log2 of the entry pairs per row (ms / 2)
    const int hp = 1 << lg;
    for (int e = threadIdx.x; e < C * hp; e += blockDim.x) {
        const int r = e >> lg, j = e & (hp - 1);
        const float sc = sbeta[r] * scale_of(r);
        if (j == 0) {
            sA[r * ld] = sc * sl.inv_sqrt_m;
            sA[r * ld + 2 * hp - 1] = 0.f;
        } else if (j <= sl.npair) {
            float s, c;
            sincospif(phase_pi_m(slam[r], j, sl), &s, &c);
            const float w = sc * sl.sqrt2_over_m;
            sA[r * ld + 2 * j - 1] = w * c;
            sA[r * ld + 2 * j] = -w * s;
        } else {
            sA[r * ld + 2 * j - 1] = 0.f;
            sA[r * ld + 2 * j] = 0.f;
        }
    }
}

// Register-tiled SIMT product for a 256-thread block seen as 16 x 16 threads:
// acc[i][j] += sum_k A(ty + 16 i, k) * B(k, tx + 16 j).
template <int TM, int TN, class FA, class FB>
__device__ __forceinline__ void simt_mm(float (&acc)[TM][TN], int K, const FA& fa, const FB& fb) {
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
#pragma unroll 4
    for (int kk = 0; kk < K; ++kk) {
        float a[TM], b[TN];
#pragma unroll
        for (int i = 0; i < TM; ++i) a[i] = fa(ty + 16 * i, kk);
#pragma unroll
        for (int j = 0; j < TN; ++j) b[j] = fb(kk, tx + 16 * j);
#pragma unroll
        for (int i = 0; i < TM; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
}

template <int TM, int TN>
__device__ __forceinline__ void zero_acc(float (&acc)[TM][TN]) {
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}
__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
    return x;
}
// Sum over the 16 threads that share ty in the 16 x 16 layout (a half warp).
__device__ __forceinline__ float half_warp_sum(float x) {
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__device__ __forceinline__ float half_warp_max(float x) {
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
    return x;
}

__device__ __forceinline__ float sigmoidf_(float x) { return 1.f / (1.f + expf(-x)); }
__device__ __forceinline__ float softplusf_(float x) { return x > 20.f ? x : log1pf(expf(x)); }

}  // namespace cyfa
