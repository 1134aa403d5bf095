// Shared-memory tile helpers of the SIMT chunk kernels (forward and backward).
#pragma once

#include "common.cuh"
#include "kernels.h"

namespace cyfa {

constexpr int LD = 129;   // padded row stride of [C][128] shared tiles

// ---------------------------------------------------------------------------------------
// Token-wise middle readout for rows r < C of sX (row stride MSZ + 1, in place):
// o'' = U(-lam) M^T softmax(M U(lam) o') with M = R Phi ([MSZ][MSZ]); the padding logits
// (slots m..MSZ-1) are excluded from the softmax and o''[m..MSZ-1] are 0.  One warp per row; swarp
// holds 2 x MSZ floats of scratch per warp.
template <int MSZ>
static __device__ __noinline__ void middle_rows(float* sX, const float* slam, int C, const float* M, const float* MT,
                            float* swarp, const Slots& sl) {
    constexpr int LDM = MSZ + 1, NP = MSZ / 64, NE = MSZ / 32, NPAIRS = MSZ / 2 - 1;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float* z = swarp + warp * 2 * MSZ;
    float* p = z + MSZ;
    for (int r = warp; r < C; r += 8) {
        float* x = sX + r * LDM;
        const float lam = slam[r];
        float cs[NP], sn[NP];
#pragma unroll
        for (int u = 0; u < NP; ++u) {
            const int j = lane + 1 + 32 * u;
            cs[u] = 1.f;
            sn[u] = 0.f;
            if (j <= sl.npair) {
                sincospif(phase_pi_m(lam, j, sl), &sn[u], &cs[u]);
                const float xc = x[2 * j - 1], xs = x[2 * j];
                z[2 * j - 1] = cs[u] * xc - sn[u] * xs;
                z[2 * j] = sn[u] * xc + cs[u] * xs;
            } else if (j <= NPAIRS) {   // padding slots (zero)
                z[2 * j - 1] = 0.f;
                z[2 * j] = 0.f;
            }
        }
        if (lane == 0) {
            z[0] = x[0];
            z[MSZ - 1] = 0.f;
        }
        __syncwarp();
        float l[NE];
#pragma unroll
        for (int u = 0; u < NE; ++u) l[u] = 0.f;
        for (int k = 0; k < MSZ; ++k) {
            const float zk = z[k];
#pragma unroll
            for (int u = 0; u < NE; ++u) l[u] = fmaf(MT[k * MSZ + lane + 32 * u], zk, l[u]);
        }
        float mx = -INFINITY;
#pragma unroll
        for (int u = 0; u < NE; ++u) {
            if (lane + 32 * u >= sl.m) l[u] = -INFINITY;
            mx = fmaxf(mx, l[u]);
        }
        mx = warp_max(mx);
        float e[NE], sum = 0.f;
#pragma unroll
        for (int u = 0; u < NE; ++u) {
            e[u] = expf(l[u] - mx);
            sum += e[u];
        }
        sum = warp_sum(sum);
        const float inv = 1.f / sum;
#pragma unroll
        for (int u = 0; u < NE; ++u) p[lane + 32 * u] = e[u] * inv;
        __syncwarp();
        float y[NE];
#pragma unroll
        for (int u = 0; u < NE; ++u) y[u] = 0.f;
        for (int i = 0; i < sl.m; ++i) {
            const float pi = p[i];
#pragma unroll
            for (int u = 0; u < NE; ++u) y[u] = fmaf(M[i * MSZ + lane + 32 * u], pi, y[u]);
        }
        __syncwarp();
#pragma unroll
        for (int u = 0; u < NE; ++u) z[lane + 32 * u] = y[u];
        __syncwarp();
#pragma unroll
        for (int u = 0; u < NP; ++u) {
            const int j = lane + 1 + 32 * u;
            if (j <= sl.npair) {
                const float yc = z[2 * j - 1], ys = z[2 * j];
                x[2 * j - 1] = cs[u] * yc + sn[u] * ys;
                x[2 * j] = -sn[u] * yc + cs[u] * ys;
            } else if (j <= NPAIRS) {
                x[2 * j - 1] = 0.f;
                x[2 * j] = 0.f;
            }
        }
        if (lane == 0) {
            x[0] = z[0];
            x[MSZ - 1] = 0.f;
        }
        __syncwarp();
    }
}

// g_cum is local to the caller's chunks of s.Cg tokens; a kernel walking shorter chunks of C
// tokens (C divides Cg) rebases it to its own chunk start by subtracting the value just before.
__device__ __forceinline__ float g_base(const Shape& s, const float* g, int b, int h, int t0,
                                        int C) {
    return (s.Cg != C && (t0 % s.Cg) != 0) ? g[((size_t)b * s.T + t0 - 1) * s.H + h] : 0.f;
}

__device__ __forceinline__ void load_gates(const Shape& s, const float* lam, const float* g,
                                           const float* beta, int b, int h, int t0, int C,
                                           float* slam, float* sg, float* sbeta) {
    const float gb = g_base(s, g, b, h, t0, C);
    for (int r = threadIdx.x; r < C; r += blockDim.x) {
        const size_t gi = ((size_t)b * s.T + t0 + r) * s.H + h;
        slam[r] = lam[gi];
        sg[r] = g[gi] - gb;
        sbeta[r] = beta[gi];
    }
}

// Stage rows [r0, r0+nr) x columns [c0, c0+32) of a [B,T,H,D] tensor into dst[r][33].
template <typename TI>
__device__ __forceinline__ void stage_tok(float* dst, const TI* X, const Shape& s, int b, int h,
                                          int t0, int nr, int c0, float mul) {
    for (int e = threadIdx.x; e < nr * 32; e += blockDim.x) {
        const int r = e >> 5, cc = e & 31;
        dst[r * 33 + cc] = mul * ldf(X, (((size_t)b * s.T + t0 + r) * s.H + h) * s.D + c0 + cc);
    }
}

}  // namespace cyfa
