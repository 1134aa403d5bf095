// Shared-memory tile helpers of the SIMT chunk kernels (forward and backward).
#pragma once

#include "../../include/cyfa.h"
#include "common.cuh"
#include "kernels.h"

namespace cyfa {

// The chunk kernels run 256 threads per block.
constexpr int SIMT_THREADS = 256;

// Launch check of the chunk kernels, at entry: the block has SIMT_THREADS threads (the staging
// and the 16 x 16 thread tiles assume it) and the dynamic shared memory covers the kernel's
// carve-up [smem, end).  A launch that does not fit records CYFA_ERR_CUDA in the translation
// unit's error word (returned by cyfa_check) and every thread leaves before touching memory.
static __device__ int g_simt_err;
__device__ __forceinline__ bool launch_ok(const float* smem, const float* end) {
    unsigned dyn;
    asm volatile("mov.u32 %0, %%dynamic_smem_size;" : "=r"(dyn));
    const bool ok = blockDim.x == SIMT_THREADS && blockDim.y == 1 && blockDim.z == 1 &&
                    (size_t)(end - smem) * sizeof(float) <= (size_t)dyn;
    if (!ok && threadIdx.x == 0) atomicExch(&g_simt_err, CYFA_ERR_CUDA);
    return ok;
}
// Reads (and clears) this translation unit's error word; synchronises the stream.
static inline cudaError_t read_simt_error(cudaStream_t st, int* err) {
    cudaError_t e = cudaMemcpyFromSymbolAsync(err, g_simt_err, sizeof(int), 0,
                                              cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return e;
    e = cudaStreamSynchronize(st);
    if (e == cudaSuccess && *err) {
        const int zero = 0;
        e = cudaMemcpyToSymbol(g_simt_err, &zero, sizeof(int));
    }
    return e;
}

// ---------------------------------------------------------------------------------------
// Token-wise middle readout for rows r < C of sX (row stride MSZ + 1, in place):
// o'' = U(-lam) M^T softmax(M U(lam) o') with M = R Phi ([MSZ][MSZ], global); the padding
// logits (slots m..MSZ-1) are excluded from the softmax and o''[m..MSZ-1] are 0.
// Each warp takes RB rows at a time so that every entry of M and M^T it loads serves RB rows.
// A lane keeps the rotation pairs j = lane + 1 + 32 u of its rows in registers and the logit /
// softmax entries lane + 32 v; the products over slots broadcast the summed-over vector from
// its owner lane by shuffles, in slot order (the same order of accumulation as a plain loop).
// C is a multiple of 8 RB.
template <int MSZ, int RB>
static __device__ __noinline__ void middle_rows(float* sX, const float* slam, int C, const float* M,
                                                const float* MT, const Slots& sl) {
    constexpr int LDM = MSZ + 1, NP = MSZ / 64, NE = MSZ / 32;
    constexpr int UNR = MSZ == 128 ? 4 : 1;   // slot steps whose M / M^T loads are in flight together
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int npair = sl.npair, m = sl.m;
    for (int r0 = warp * RB; r0 < C; r0 += 8 * RB) {
        float cs[RB][NP], sn[RB][NP], zc[RB][NP], zs[RB][NP], z0[RB];
#pragma unroll
        for (int rb = 0; rb < RB; ++rb) {
            const float* x = sX + (r0 + rb) * LDM;
            const float lam = slam[r0 + rb];
            z0[rb] = x[0];
#pragma unroll
            for (int u = 0; u < NP; ++u) {
                const int j = lane + 1 + 32 * u;
                cs[rb][u] = 1.f;
                sn[rb][u] = 0.f;
                zc[rb][u] = zs[rb][u] = 0.f;
                if (j <= npair) {   // z = U(lam) o'
                    sincospif(phase_pi_m(lam, j, sl), &sn[rb][u], &cs[rb][u]);
                    const float xc = x[2 * j - 1], xs = x[2 * j];
                    zc[rb][u] = cs[rb][u] * xc - sn[rb][u] * xs;
                    zs[rb][u] = sn[rb][u] * xc + cs[rb][u] * xs;
                }
            }
        }
        // logits l[col] = sum_k MT[k][col] z[k], col = lane + 32 v
        float l[RB][NE];
#pragma unroll
        for (int v = 0; v < NE; ++v) {
            const float mt = MT[lane + 32 * v];
#pragma unroll
            for (int rb = 0; rb < RB; ++rb) l[rb][v] = mt * z0[rb];
        }
#pragma unroll
        for (int u = 0; u < NP; ++u) {
            const int jmax = min(32, npair - 32 * u);   // pairs 32 u + 1 .. 32 u + jmax
#pragma unroll UNR
            for (int src = 0; src < jmax; ++src) {
                const int kc = 2 * (32 * u + src) + 1;
                float vc[RB], vs[RB];
#pragma unroll
                for (int rb = 0; rb < RB; ++rb) {
                    vc[rb] = __shfl_sync(0xffffffffu, zc[rb][u], src);
                    vs[rb] = __shfl_sync(0xffffffffu, zs[rb][u], src);
                }
                const float* mc = MT + kc * MSZ + lane;
#pragma unroll
                for (int v = 0; v < NE; ++v) {
                    const float a = mc[32 * v], b = mc[MSZ + 32 * v];
#pragma unroll
                    for (int rb = 0; rb < RB; ++rb)
                        l[rb][v] = fmaf(b, vs[rb], fmaf(a, vc[rb], l[rb][v]));
                }
            }
        }
        // softmax over the m active slots
#pragma unroll
        for (int rb = 0; rb < RB; ++rb) {
            float mx = -INFINITY;
#pragma unroll
            for (int v = 0; v < NE; ++v) {
                if (lane + 32 * v >= m) l[rb][v] = -INFINITY;
                mx = fmaxf(mx, l[rb][v]);
            }
            mx = warp_max(mx);
            float sum = 0.f;
#pragma unroll
            for (int v = 0; v < NE; ++v) {
                l[rb][v] = expf(l[rb][v] - mx);
                sum += l[rb][v];
            }
            const float inv = 1.f / warp_sum(sum);
#pragma unroll
            for (int v = 0; v < NE; ++v) l[rb][v] *= inv;
        }
        // y[col] = sum_{i < m} M[i][col] p[i], into the row (o' is consumed)
        float y[RB][NE];
#pragma unroll
        for (int rb = 0; rb < RB; ++rb)
#pragma unroll
            for (int v = 0; v < NE; ++v) y[rb][v] = 0.f;
#pragma unroll
        for (int v2 = 0; v2 < NE; ++v2) {
            const int imax = min(32, m - 32 * v2);
#pragma unroll UNR
            for (int src = 0; src < imax; ++src) {
                float pv[RB];
#pragma unroll
                for (int rb = 0; rb < RB; ++rb) pv[rb] = __shfl_sync(0xffffffffu, l[rb][v2], src);
                const float* mr = M + (32 * v2 + src) * MSZ + lane;
#pragma unroll
                for (int v = 0; v < NE; ++v) {
                    const float a = mr[32 * v];
#pragma unroll
                    for (int rb = 0; rb < RB; ++rb) y[rb][v] = fmaf(a, pv[rb], y[rb][v]);
                }
            }
        }
        __syncwarp();
#pragma unroll
        for (int rb = 0; rb < RB; ++rb) {
            float* x = sX + (r0 + rb) * LDM;
#pragma unroll
            for (int v = 0; v < NE; ++v) x[lane + 32 * v] = y[rb][v];   // padding entries are 0
        }
        __syncwarp();
#pragma unroll
        for (int rb = 0; rb < RB; ++rb) {   // o'' = U(-lam) y on the active pairs
            float* x = sX + (r0 + rb) * LDM;
#pragma unroll
            for (int u = 0; u < NP; ++u) {
                const int j = lane + 1 + 32 * u;
                if (j <= npair) {
                    const float yc = x[2 * j - 1], ys = x[2 * j];
                    x[2 * j - 1] = cs[rb][u] * yc + sn[rb][u] * ys;
                    x[2 * j] = -sn[rb][u] * yc + cs[rb][u] * ys;
                }
            }
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

// Staging of `count` elements by the block: thread t moves e = t + 256 k (k < PER, e < count)
// with ld(e) -> st(e, value).  Each thread issues all its loads before its first store, so its
// global loads are in flight together (a load-store loop would wait out a full memory latency
// per element: the compiler cannot move a load past a store that may alias it).
template <int PER, class Ld, class St>
__device__ __forceinline__ void stage_elems(int count, const Ld& ld, const St& st) {
    float v[PER];
#pragma unroll
    for (int k = 0; k < PER; ++k) {
        const int e = threadIdx.x + SIMT_THREADS * k;
        v[k] = e < count ? ld(e) : 0.f;
    }
#pragma unroll
    for (int k = 0; k < PER; ++k) {
        const int e = threadIdx.x + SIMT_THREADS * k;
        if (e < count) st(e, v[k]);
    }
}

// Stage rows [t0, t0+NR) x columns [c0, c0+NC) of a [B,T,H,D] tensor into dst[r][NC + 1].
template <int NR, int NC = 32, typename TI>
__device__ __forceinline__ void stage_tok(float* dst, const TI* X, const Shape& s, int b, int h,
                                          int t0, int c0, float mul) {
    static_assert(NR * NC % SIMT_THREADS == 0, "rows x columns in whole passes of the block");
    stage_elems<NR * NC / SIMT_THREADS>(
        NR * NC,
        [&](int e) {
            return mul * ldf(X, (((size_t)b * s.T + t0 + e / NC) * s.H + h) * s.D + c0 + e % NC);
        },
        [&](int e, float x) { dst[(e / NC) * (NC + 1) + e % NC] = x; });
}

}  // namespace cyfa
