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

// Row blocks times a global matrix: acc[p][i][j] += sum_{k < K} X_p(ty + 16 i, k) B(k, tx + 16 j)
// for p < NPROD (X_0, X_1 rows in shared memory with stride MSZ + 1; X_1 unused when NPROD = 1)
// and B a [MSZ][MSZ] global matrix whose rows are staged 32 at a time through sB
// ([32][MSZ + 1]): one staging of B serves every product.  K is a multiple of 32, at most MSZ.
// Begins with a block barrier; the caller places one before sB or the X rows are rewritten.
template <int NPROD, int TM, int MSZ>
__device__ __forceinline__ void rows_times_gmat(float (&acc)[NPROD][TM][MSZ / 16], float* sB,
                                                const float* X0, const float* X1, const float* B,
                                                int K) {
    constexpr int LDM = MSZ + 1, NJ = MSZ / 16;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    for (int k0 = 0; k0 < K; k0 += 32) {
        __syncthreads();
        stage_elems<32 * MSZ / SIMT_THREADS>(
            32 * MSZ, [&](int e) { return B[(size_t)k0 * MSZ + e]; },
            [&](int e, float x) { sB[(e / MSZ) * LDM + e % MSZ] = x; });
        __syncthreads();
#pragma unroll 2
        for (int kk = 0; kk < 32; ++kk) {
            float a[NPROD][TM], b[NJ];
#pragma unroll
            for (int i = 0; i < TM; ++i) {
                a[0][i] = X0[(ty + 16 * i) * LDM + k0 + kk];
                if (NPROD > 1) a[NPROD - 1][i] = X1[(ty + 16 * i) * LDM + k0 + kk];
            }
#pragma unroll
            for (int j = 0; j < NJ; ++j) b[j] = sB[kk * LDM + tx + 16 * j];
#pragma unroll
            for (int p = 0; p < NPROD; ++p)
#pragma unroll
                for (int i = 0; i < TM; ++i)
#pragma unroll
                    for (int j = 0; j < NJ; ++j) acc[p][i][j] = fmaf(a[p][i], b[j], acc[p][i][j]);
        }
    }
}

// The middle readout for the C rows of a chunk (o' in the rows of sX, stride MSZ + 1, replaced by
// o''), as products of the row block with M^T and M (global [MSZ][MSZ], zero beyond the m active
// rows and columns): z = U(lam) o' (in place; inactive entries zeroed), l = M z (one pass over
// M^T), p = softmax(l) over the m active slots (into sX), y = M^T p (one pass over M, into sX),
// o'' = U(-lam) y.  The row ty + 16 i of a product lives on the 16 threads of a half warp.  sB is
// the [32][MSZ + 1] staging of M^T and M.  Needs a block barrier before (o' complete) and after.
template <int C, int MSZ>
static __device__ __noinline__ void readout_rows_fwd(float* sX, float* sB, const float* slam,
                                                     const float* M, const float* MT,
                                                     const Slots& sl) {
    constexpr int LDM = MSZ + 1, NP = MSZ / 64, TM = C / 16, NJ = MSZ / 16, NW = SIMT_THREADS / 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int npair = sl.npair, m = sl.m;
    const int K = (m + 31) & ~31;   // the products run over the active entries in steps of 32
    for (int r = warp; r < C; r += NW) {
        float* z = sX + r * LDM;
        const float lam = slam[r];
#pragma unroll
        for (int u = 0; u < NP; ++u) {
            const int j = lane + 1 + 32 * u;
            if (j <= npair) {
                float sn, cs;
                sincospif(phase_pi_m(lam, j, sl), &sn, &cs);
                const float xc = z[2 * j - 1], xs = z[2 * j];
                z[2 * j - 1] = cs * xc - sn * xs;
                z[2 * j] = sn * xc + cs * xs;
            } else if (j < MSZ / 2) {
                z[2 * j - 1] = z[2 * j] = 0.f;
            }
        }
        if (lane == 0) z[MSZ - 1] = 0.f;
    }
    float acc[1][TM][NJ];
    zero_acc(acc[0]);
    rows_times_gmat<1, TM, MSZ>(acc, sB, sX, sX, MT, K);
#pragma unroll
    for (int i = 0; i < TM; ++i) {
        float mx = -INFINITY;
#pragma unroll
        for (int j = 0; j < NJ; ++j)
            if (tx + 16 * j < m) mx = fmaxf(mx, acc[0][i][j]);
        mx = half_warp_max(mx);
        float sum = 0.f;
#pragma unroll
        for (int j = 0; j < NJ; ++j) {
            acc[0][i][j] = tx + 16 * j < m ? expf(acc[0][i][j] - mx) : 0.f;
            sum += acc[0][i][j];
        }
        const float inv = 1.f / half_warp_sum(sum);
#pragma unroll
        for (int j = 0; j < NJ; ++j) acc[0][i][j] *= inv;
    }
    __syncthreads();   // z has been read
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < NJ; ++j) sX[(ty + 16 * i) * LDM + tx + 16 * j] = acc[0][i][j];
    zero_acc(acc[0]);
    rows_times_gmat<1, TM, MSZ>(acc, sB, sX, sX, M, K);
    __syncthreads();   // p has been read
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < NJ; ++j) sX[(ty + 16 * i) * LDM + tx + 16 * j] = acc[0][i][j];
    __syncthreads();
    for (int r = warp; r < C; r += NW) {   // o'' = U(-lam) y on the active pairs
        float* x = sX + r * LDM;
        const float lam = slam[r];
#pragma unroll
        for (int u = 0; u < NP; ++u) {
            const int j = lane + 1 + 32 * u;
            if (j <= npair) {
                float sn, cs;
                sincospif(phase_pi_m(lam, j, sl), &sn, &cs);
                const float yc = x[2 * j - 1], ys = x[2 * j];
                x[2 * j - 1] = cs * yc + sn * ys;
                x[2 * j] = -sn * yc + cs * ys;
            }
        }
    }
}

}  // namespace cyfa
