// The operator's neighbours inside the CyFA mixer (Sec. 3.4, Mixer and backbone), as the memory-
// bound kernels around the chunk calls:
//   before: ShortConv over tokens (causal, depthwise, width K = 4, zero history) + SiLU on the
//           projected q, k, v, then RMSNorm over the head dimension on q and k (gain g shared by
//           the heads):  a_t = silu(sum_i w_i x_{t-3+i}),  q_t = a_t / sqrt(mean(a_t^2) + eps) * g;
//   after:  head-wise RMSNorm of the operator output times a sigmoid gate whose logits z come
//           from the mixer's low-rank gate projection:  y_t = o_t / sqrt(mean(o_t^2) + eps) * g *
//           sigmoid(z_t);
// and their backward passes.  The paper states these layers without formulas; the width, the
// activation and the gain sharing are this library's reading.
//
// Layout: every tensor is [B, T, H, d] (bf16 or fp32), channel c = h d + i; filters [H d][4] fp32;
// gains [d] fp32.  d / 8 lanes per (token, head) row, eight consecutive channels per lane
// (16-byte accesses).  The ShortConv kernels give each thread a range of tokens of one head and
// keep the last rows of x in registers (one HBM read per element, no shared memory); the row
// kernels (post) walk rows grid-stride.  Parameter gradients (filters, gains) are summed per
// block in registers and written as partials, then reduced by a second kernel (deterministic).
#include <type_traits>

#include "../../include/cyfa.h"
#include "common.cuh"
#include "kernels.h"

namespace cyfa {

namespace {

constexpr int KW = 4;        // ShortConv width
constexpr int TT = 64;       // tokens per tile
constexpr int NW = 8;        // warps per block

// sigmoid with the fast exponential and divide intrinsics (relative error ~1e-6, far below the
// bf16 rounding of every output); the argument is clamped so the divisor stays below 2^126
__device__ __forceinline__ float sigm_(float u) {
    return __fdividef(1.f, 1.f + __expf(-fmaxf(u, -80.f)));
}
__device__ __forceinline__ float silu_(float u) { return u * sigm_(u); }

// Eight consecutive elements of a bf16 / fp32 tensor <-> eight floats (one 16-byte access for
// bf16, two for fp32; the element offset is a multiple of 8).
__device__ __forceinline__ void ld8(const __nv_bfloat16* p, float (&x)[8]) {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float2 f = __bfloat1622float2(h[j]);
        x[2 * j] = f.x;
        x[2 * j + 1] = f.y;
    }
}
__device__ __forceinline__ void ld8(const float* p, float (&x)[8]) {
    const float4 a = *reinterpret_cast<const float4*>(p), b = *reinterpret_cast<const float4*>(p + 4);
    x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w; x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
}
__device__ __forceinline__ void st8(__nv_bfloat16* p, const float (&x)[8]) {
    uint4 u;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
    for (int j = 0; j < 4; ++j) h[j] = __floats2bfloat162_rn(x[2 * j], x[2 * j + 1]);
    *reinterpret_cast<uint4*>(p) = u;
}
__device__ __forceinline__ void st8(float* p, const float (&x)[8]) {
    *reinterpret_cast<float4*>(p) = make_float4(x[0], x[1], x[2], x[3]);
    *reinterpret_cast<float4*>(p + 4) = make_float4(x[4], x[5], x[6], x[7]);
}
// shared memory (16-byte aligned) <-> eight floats
__device__ __forceinline__ void lds8(const float* p, float (&x)[8]) { ld8(p, x); }
__device__ __forceinline__ void sts8(float* p, const float (&x)[8]) { st8(p, x); }

// Sum over the LPR lanes that hold one row (aligned groups of LPR lanes, LPR a power of two).
template <int LPR>
__device__ __forceinline__ float row_sum(float x) {
#pragma unroll
    for (int o = LPR / 2; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

struct PreArgs {
    Shape s;
    const void* x[3];        // projected q, k, v (ShortConv inputs)
    const float* w[3];       // filters [H*d][KW]
    const float* g[2];       // RMSNorm gains of q, k [d]
    float eps;
    void* y[3];              // outputs
    // backward
    const void* dy[3];
    void* dx[3];
    float* dw_part;          // [3][nsplit * B][H*d][KW]
    float* dg_part;          // [2][nsplit * B * H][d]
    int nsplit;
};

// Lane roles in the row kernels (post): LPR = d / 8 lanes per row, 8 consecutive channels per
// lane, RPW rows per warp at a time.
template <int D>
struct Roles {
    static constexpr int LPR = D / 8, RPW = 32 / LPR, RPB = RPW * NW;
    int sub, c0;
    __device__ Roles() {
        const int lane = threadIdx.x & 31;
        sub = lane / LPR;
        c0 = (lane % LPR) * 8;
    }
};

// N consecutive elements (N = 4 or 8; the offset a multiple of N) of a bf16 / fp32 tensor as
// loaded, converted to floats on use: bf16 in one 8- or 16-byte word, fp32 in N floats.
template <typename TI, int N> struct RawN;
template <int N> struct RawN<__nv_bfloat16, N> {
    using W = typename std::conditional<N == 8, uint4, uint2>::type;
    W u;
    __device__ void load(const __nv_bfloat16* p) { u = *reinterpret_cast<const W*>(p); }
    __device__ void zero() { u = W{}; }
    __device__ void get(float (&x)[N]) const {
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
        for (int j = 0; j < N / 2; ++j) {
            const float2 f = __bfloat1622float2(h[j]);
            x[2 * j] = f.x;
            x[2 * j + 1] = f.y;
        }
    }
};
template <int N> struct RawN<float, N> {
    float v[N];
    __device__ void load(const float* p) {
#pragma unroll
        for (int j = 0; j < N; j += 4) {
            const float4 f = *reinterpret_cast<const float4*>(p + j);
            v[j] = f.x; v[j + 1] = f.y; v[j + 2] = f.z; v[j + 3] = f.w;
        }
    }
    __device__ void zero() {
#pragma unroll
        for (int j = 0; j < N; ++j) v[j] = 0.f;
    }
    __device__ void get(float (&x)[N]) const {
#pragma unroll
        for (int j = 0; j < N; ++j) x[j] = v[j];
    }
};
template <int N>
__device__ __forceinline__ void stN(__nv_bfloat16* p, const float (&x)[N]) {
    using W = typename std::conditional<N == 8, uint4, uint2>::type;
    W u;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
    for (int j = 0; j < N / 2; ++j) h[j] = __floats2bfloat162_rn(x[2 * j], x[2 * j + 1]);
    *reinterpret_cast<W*>(p) = u;
}
template <int N>
__device__ __forceinline__ void stN(float* p, const float (&x)[N]) {
#pragma unroll
    for (int j = 0; j < N; j += 4)
        *reinterpret_cast<float4*>(p + j) = make_float4(x[j], x[j + 1], x[j + 2], x[j + 3]);
}

// Lane roles in the ShortConv kernels: N = 4 channels per thread (8 at d = 256), so that a head
// row spans LPR = d / N <= 32 consecutive lanes of one warp; a block of 256 threads covers
// HB = 256 / LPR heads of one batch row and one tensor.  Each thread walks a range of tokens of
// its head, keeping the last rows of x in registers: every element of x is read from HBM once,
// with no shared memory and no block barrier.
template <int D>
struct ConvRoles {
    static constexpr int N = D <= 128 ? 4 : 8, LPR = D / N, HB = 256 / LPR;
    int hl, c0;
    __device__ ConvRoles() {
        hl = threadIdx.x / LPR;
        c0 = (threadIdx.x % LPR) * N;
    }
};

// Row (b, t, h) of a [B, T, H, d] tensor as loaded, zero unless 0 <= t < tend (tend <= T) and
// h < H.
template <int D, typename TI, int N>
__device__ __forceinline__ void ld_raw(const TI* X, int T, int tend, int H, int b, int t, int h,
                                       int c0, RawN<TI, N>& r) {
    if (t >= 0 && t < tend && h < H) r.load(X + (((size_t)b * T + t) * H + h) * D + c0);
    else r.zero();
}

constexpr int UF = 4;    // tokens whose loads are issued together (forward)
constexpr int UB = 4;    // the same in the backward

// Forward: grid (ceil(H / HB), nsplit, 3 B); block 256.
template <int D, typename TI>
__global__ void __launch_bounds__(256, D <= 128 ? 4 : 1) mixer_pre_kernel(PreArgs a) {
    using R = ConvRoles<D>;
    constexpr int N = R::N;
    const R ro;
    const int H = a.s.H, T = a.s.T, B = a.s.B;
    const int h = blockIdx.x * R::HB + ro.hl, sp = blockIdx.y;
    const int z = blockIdx.z / B, b = blockIdx.z % B;
    const bool hv = h < H;
    const TI* X = (const TI*)a.x[z];
    TI* Y = (TI*)a.y[z];
    float w[KW][N], gain[N];
#pragma unroll
    for (int j = 0; j < N; ++j) {
        gain[j] = z < 2 ? a.g[z][ro.c0 + j] : 1.f;
#pragma unroll
        for (int k = 0; k < KW; ++k) w[k][j] = hv ? a.w[z][((size_t)h * D + ro.c0 + j) * KW + k] : 0.f;
    }
    const int per = (T + a.nsplit - 1) / a.nsplit;
    const int tb = sp * per, te = min(T, tb + per);
    float ring[KW - 1][N];    // x rows t - 3, t - 2, t - 1
#pragma unroll
    for (int k = 0; k < KW - 1; ++k) {
        RawN<TI, N> r;
        ld_raw<D>(X, T, T, H, b, tb - (KW - 1) + k, h, ro.c0, r);
        r.get(ring[k]);
    }
    for (int t0 = tb; t0 < te; t0 += UF) {
        RawN<TI, N> xraw[UF];
#pragma unroll
        for (int u = 0; u < UF; ++u) ld_raw<D>(X, T, te, H, b, t0 + u, h, ro.c0, xraw[u]);
#pragma unroll
        for (int u = 0; u < UF; ++u) {
            float v[N], xu[N], ss = 0.f;
            xraw[u].get(xu);
#pragma unroll
            for (int j = 0; j < N; ++j) {
                float acc = w[KW - 1][j] * xu[j];
#pragma unroll
                for (int k = 0; k < KW - 1; ++k) acc = fmaf(w[k][j], ring[k][j], acc);
                v[j] = silu_(acc);
                ss = fmaf(v[j], v[j], ss);
            }
            ss = row_sum<R::LPR>(ss);   // all lanes of the warp run the same tokens
            const float rr = z < 2 ? rsqrtf(ss * (1.f / D) + a.eps) : 1.f;
#pragma unroll
            for (int j = 0; j < N; ++j) {
                v[j] *= rr * gain[j];
#pragma unroll
                for (int k = 0; k < KW - 2; ++k) ring[k][j] = ring[k + 1][j];
                ring[KW - 2][j] = xu[j];
            }
            if (hv && t0 + u < te) stN<N>(Y + (((size_t)b * T + t0 + u) * H + h) * D + ro.c0, v);
        }
    }
}

// Backward: grid (ceil(H / HB), nsplit, 3 B); block 256.  Each thread walks its tokens from the
// last to the first: du_t needs x_{t-3..t} (a ring refilled with x_{t-4} after each token) and
// dy_t; dx_t = sum_k w_k du_{t+3-k} needs the three du after it (a second ring, primed with the
// three tokens past the range).  Filter and gain gradients accumulate in registers.
template <int D, typename TI>
__global__ void __launch_bounds__(256, D <= 128 ? 2 : 1) mixer_pre_bwd_kernel(PreArgs a) {
    using R = ConvRoles<D>;
    constexpr int N = R::N;
    const R ro;
    const int H = a.s.H, T = a.s.T, B = a.s.B;
    const int h = blockIdx.x * R::HB + ro.hl, sp = blockIdx.y;
    const int z = blockIdx.z / B, b = blockIdx.z % B;
    const bool hv = h < H;
    const TI* X = (const TI*)a.x[z];
    const TI* DY = (const TI*)a.dy[z];
    TI* DX = (TI*)a.dx[z];
    float w[KW][N], gain[N], wacc[KW][N], gacc[N];
#pragma unroll
    for (int j = 0; j < N; ++j) {
        gain[j] = z < 2 ? a.g[z][ro.c0 + j] : 1.f;
        gacc[j] = 0.f;
#pragma unroll
        for (int k = 0; k < KW; ++k) {
            w[k][j] = hv ? a.w[z][((size_t)h * D + ro.c0 + j) * KW + k] : 0.f;
            wacc[k][j] = 0.f;
        }
    }
    const int per = (T + a.nsplit - 1) / a.nsplit;
    const int tb = sp * per, te = min(T, tb + per);
    float xr[KW][N];          // x rows t - 3 .. t (xr[3] = x_t)
    float dur[KW - 1][N];     // du rows t + 1 .. t + 3

    // du_t from the ring xr (x_{t-3..t}) and dy_t; gain partial when `own`
    auto du_of = [&](const float (&gv)[N], bool own, float (&du)[N]) {
        float av[N], sg[N], ss = 0.f, ea = 0.f;   // sg: silu'(u), from one sigmoid
#pragma unroll
        for (int j = 0; j < N; ++j) {
            float acc = 0.f;
#pragma unroll
            for (int k = 0; k < KW; ++k) acc = fmaf(w[k][j], xr[k][j], acc);
            const float sv = sigm_(acc);
            av[j] = acc * sv;
            sg[j] = sv * (1.f + acc * (1.f - sv));
            ss = fmaf(av[j], av[j], ss);
            ea = fmaf(gv[j] * gain[j], av[j], ea);
        }
        ss = row_sum<R::LPR>(ss);
        ea = row_sum<R::LPR>(ea);
        float rr = 1.f, coef = 0.f;
        if (z < 2) {
            rr = rsqrtf(ss * (1.f / D) + a.eps);
            coef = ea * rr * rr * rr * (1.f / D);
        }
#pragma unroll
        for (int j = 0; j < N; ++j) {
            const float da = z < 2 ? rr * gv[j] * gain[j] - av[j] * coef : gv[j];
            du[j] = da * sg[j];
            if (own && z < 2) gacc[j] = fmaf(gv[j], av[j] * rr, gacc[j]);
        }
    };
    // one token back: xr <- x_{t-4..t-1} given x_{t-4} in `older`
    auto x_back = [&](const float (&older)[N]) {
#pragma unroll
        for (int j = 0; j < N; ++j) {
#pragma unroll
            for (int k = KW - 1; k > 0; --k) xr[k][j] = xr[k - 1][j];
            xr[0][j] = older[j];
        }
    };

    // prime: x_{te-1..te+2}, then du of the tokens te + 2, te + 1, te (zero past T), stepping the
    // x ring back to x_{te-4..te-1}, which token te - 1 needs
    const int tp = te + KW - 2;
#pragma unroll
    for (int k = 0; k < KW; ++k) {
        RawN<TI, N> r;
        ld_raw<D>(X, T, T, H, b, tp - (KW - 1) + k, h, ro.c0, r);
        r.get(xr[k]);
    }
#pragma unroll
    for (int i = KW - 2; i >= 0; --i) {
        RawN<TI, N> rg, rx;
        ld_raw<D>(DY, T, T, H, b, te + i, h, ro.c0, rg);
        ld_raw<D>(X, T, T, H, b, te + i - KW, h, ro.c0, rx);
        float gv[N], older[N];
        rg.get(gv);
        du_of(gv, false, dur[i]);
        rx.get(older);
        x_back(older);
    }
    constexpr int U = N == 8 ? UB / 2 : UB;   // eight channels per thread hold twice the state
    for (int t1 = te; t1 > tb; t1 -= U) {
        const int n = min(U, t1 - tb);           // the same for every lane of the block
        RawN<TI, N> graw[U], xraw[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int t = t1 - 1 - u;
            ld_raw<D>(DY, T, (u < n) ? T : 0, H, b, t, h, ro.c0, graw[u]);
            ld_raw<D>(X, T, (u < n) ? T : 0, H, b, t - KW, h, ro.c0, xraw[u]);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (u >= n) break;
            const int t = t1 - 1 - u;
            float du[N], gv[N], dxv[N], xo[N];
            graw[u].get(gv);
            du_of(gv, true, du);
#pragma unroll
            for (int j = 0; j < N; ++j) {
                dxv[j] = w[KW - 1][j] * du[j];
#pragma unroll
                for (int k = 0; k < KW - 1; ++k) dxv[j] = fmaf(w[KW - 2 - k][j], dur[k][j], dxv[j]);
#pragma unroll
                for (int k = 0; k < KW; ++k) wacc[k][j] = fmaf(du[j], xr[k][j], wacc[k][j]);
#pragma unroll
                for (int k = KW - 2; k > 0; --k) dur[k][j] = dur[k - 1][j];
                dur[0][j] = du[j];
            }
            if (hv) stN<N>(DX + (((size_t)b * T + t) * H + h) * D + ro.c0, dxv);
            xraw[u].get(xo);
            x_back(xo);
        }
    }
    // partials of this (split, b, h)
    if (hv) {
        const size_t row = (size_t)sp * B + b;
        float* dwp = a.dw_part + (((size_t)z * a.nsplit * B + row) * H + h) * D * KW;
#pragma unroll
        for (int j = 0; j < N; ++j)
#pragma unroll
            for (int k = 0; k < KW; ++k) dwp[(ro.c0 + j) * KW + k] = wacc[k][j];
        if (z < 2) stN<N>(a.dg_part + (((size_t)z * a.nsplit * B + row) * H + h) * D + ro.c0, gacc);
    }
}

// Sums of the partials: dw[z][c][k] over the nsplit * B rows; dg[z][i] over rows and heads.
__global__ void __launch_bounds__(256) mixer_pre_reduce_kernel(PreArgs a, float* dw0, float* dw1,
                                                               float* dw2, float* dg0, float* dg1) {
    const int z = blockIdx.y, D = a.s.D, H = a.s.H, nrow = a.nsplit * a.s.B;
    float* dw = z == 0 ? dw0 : z == 1 ? dw1 : dw2;
    const size_t nw = (size_t)H * D * KW;
    for (size_t e = (size_t)blockIdx.x * blockDim.x + threadIdx.x; e < nw;
         e += (size_t)gridDim.x * blockDim.x) {
        double acc = 0.0;
        for (int r = 0; r < nrow; ++r) acc += a.dw_part[((size_t)z * nrow + r) * nw + e];
        dw[e] = (float)acc;
    }
    if (z < 2 && blockIdx.x == 0) {
        float* dg = z == 0 ? dg0 : dg1;
        for (int i = threadIdx.x; i < D; i += blockDim.x) {
            double acc = 0.0;
            for (int r = 0; r < nrow * H; ++r) acc += a.dg_part[((size_t)z * nrow * H + r) * D + i];
            dg[i] = (float)acc;
        }
    }
}

struct PostArgs {
    Shape s;
    const void *o, *zl;     // operator output, gate logits
    const float* g;         // gain [d]
    float eps;
    void* y;
    const void* dy;
    void *dO, *dz;
    float* dg_part;         // [nblock][d]
};

// One row group (d / 8 lanes) per (token, head) row, RPW rows per warp; grid-stride over rows.
template <int D, typename TI>
__global__ void __launch_bounds__(256) mixer_post_kernel(PostArgs a) {
    using R = Roles<D>;
    const R ro;
    const size_t rows = (size_t)a.s.B * a.s.T * a.s.H;
    const TI* O = (const TI*)a.o;
    const TI* Z = (const TI*)a.zl;
    TI* Y = (TI*)a.y;
    float gain[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) gain[j] = a.g[ro.c0 + j];
    const size_t stride = (size_t)gridDim.x * R::RPB;
    // trip counts agree across a warp (rows of one warp are consecutive), so the shuffles are
    // never split
    for (size_t r0 = (size_t)blockIdx.x * R::RPB + (threadIdx.x >> 5) * R::RPW; r0 < rows;
         r0 += stride) {
        const size_t row = r0 + ro.sub;
        const bool live = row < rows;
        float ov[8], zv[8];
        if (live) {
            ld8(O + row * D + ro.c0, ov);
            ld8(Z + row * D + ro.c0, zv);
        } else {
#pragma unroll
            for (int j = 0; j < 8; ++j) ov[j] = zv[j] = 0.f;
        }
        float ss = 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j) ss = fmaf(ov[j], ov[j], ss);
        const float rr = rsqrtf(row_sum<R::LPR>(ss) * (1.f / D) + a.eps);
#pragma unroll
        for (int j = 0; j < 8; ++j) ov[j] = ov[j] * rr * gain[j] * sigm_(zv[j]);
        if (live) st8(Y + row * D + ro.c0, ov);
    }
}

template <int D, typename TI>
__global__ void __launch_bounds__(256) mixer_post_bwd_kernel(PostArgs a) {
    using R = Roles<D>;
    const R ro;
    const int warp = threadIdx.x >> 5;
    const size_t rows = (size_t)a.s.B * a.s.T * a.s.H;
    const TI* O = (const TI*)a.o;
    const TI* Z = (const TI*)a.zl;
    const TI* DYp = (const TI*)a.dy;
    TI* DO = (TI*)a.dO;
    TI* DZ = (TI*)a.dz;
    float gain[8], gacc[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        gain[j] = a.g[ro.c0 + j];
        gacc[j] = 0.f;
    }
    const size_t stride = (size_t)gridDim.x * R::RPB;
    for (size_t r0 = (size_t)blockIdx.x * R::RPB + warp * R::RPW; r0 < rows; r0 += stride) {
        const size_t row = r0 + ro.sub;
        const bool live = row < rows;
        float ov[8], sv[8], ev[8];
        if (live) {
            float zv[8], dyv[8];
            ld8(O + row * D + ro.c0, ov);
            ld8(Z + row * D + ro.c0, zv);
            ld8(DYp + row * D + ro.c0, dyv);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                sv[j] = sigm_(zv[j]);
                ev[j] = dyv[j] * sv[j];          // gradient reaching rms(o) * g
            }
        } else {
#pragma unroll
            for (int j = 0; j < 8; ++j) ov[j] = sv[j] = ev[j] = 0.f;
        }
        float ss = 0.f, eo = 0.f;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            ss = fmaf(ov[j], ov[j], ss);
            eo = fmaf(ev[j] * gain[j], ov[j], eo);
        }
        const float rr = rsqrtf(row_sum<R::LPR>(ss) * (1.f / D) + a.eps);
        const float coef = row_sum<R::LPR>(eo) * rr * rr * rr * (1.f / D);
        float dov[8], dzv[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const float n = ov[j] * rr;
            dov[j] = rr * ev[j] * gain[j] - ov[j] * coef;
            // dz = dy * rms(o) g * s (1 - s), with dy s = ev
            dzv[j] = ev[j] * n * gain[j] * (1.f - sv[j]);
            gacc[j] = fmaf(ev[j], n, gacc[j]);
        }
        if (live) {
            st8(DO + row * D + ro.c0, dov);
            st8(DZ + row * D + ro.c0, dzv);
        }
    }
    __shared__ __align__(16) float sg[NW * 4][256];
    sts8(&sg[warp * R::RPW + ro.sub][ro.c0], gacc);
    __syncthreads();
    for (int i = threadIdx.x; i < D; i += blockDim.x) {
        float acc = 0.f;
        for (int w = 0; w < NW * R::RPW; ++w) acc += sg[w][i];
        a.dg_part[(size_t)blockIdx.x * D + i] = acc;
    }
}

__global__ void __launch_bounds__(256) mixer_post_reduce_kernel(const float* part, int nblock,
                                                                int D, float* dg) {
    for (int i = threadIdx.x; i < D; i += blockDim.x) {
        double acc = 0.0;
        for (int r = 0; r < nblock; ++r) acc += part[(size_t)r * D + i];
        dg[i] = (float)acc;
    }
}

int post_blocks(const Shape& s) {
    const long long rows = (long long)s.B * s.T * s.H;
    const long long want = (rows + NW - 1) / NW;
    return (int)(want < 152 * 8 ? want : 152 * 8);
}

// Token splits per (batch row, head group, tensor): about eight blocks per SM in all, each
// walking at least 64 tokens (its first three rows are re-read from the previous range).
int pre_splits(const Shape& s, bool bwd) {
    const int hb = 256 / (s.D <= 128 ? s.D / 4 : s.D / 8);
    const long long groups = (long long)s.B * 3 * ((s.H + hb - 1) / hb);
    long long n = (8LL * 152 + groups - 1) / groups;
    const long long most = (s.T + 63) / 64;
    if (n > most) n = most;
    (void)bwd;
    return (int)(n < 1 ? 1 : n);
}

template <int D, typename TI>
cudaError_t pre_launch(PreArgs a, bool bwd, float* const* outs, cudaStream_t st) {
    const int hg = (a.s.H + ConvRoles<D>::HB - 1) / ConvRoles<D>::HB;
    const dim3 grid(hg, a.nsplit, 3 * a.s.B);
    if (!bwd) {
        { LaunchScope ls_("mixer_pre", st); mixer_pre_kernel<D, TI><<<grid, 256, 0, st>>>(a); }
        return cudaGetLastError();
    }
    { LaunchScope ls_("mixer_pre_bwd", st); mixer_pre_bwd_kernel<D, TI><<<grid, 256, 0, st>>>(a); }
    const int nb = (int)(((size_t)a.s.H * D * KW + 255) / 256);
    { LaunchScope ls_("mixer_pre_reduce", st);
      mixer_pre_reduce_kernel<<<dim3(nb, 3), 256, 0, st>>>(a, outs[0], outs[1], outs[2], outs[3], outs[4]); }
    return cudaGetLastError();
}

template <int D, typename TI>
cudaError_t post_launch(PostArgs a, bool bwd, float* dg, cudaStream_t st) {
    const int nb = post_blocks(a.s);
    if (!bwd) {
        { LaunchScope ls_("mixer_post", st); mixer_post_kernel<D, TI><<<nb, 256, 0, st>>>(a); }
        return cudaGetLastError();
    }
    { LaunchScope ls_("mixer_post_bwd", st); mixer_post_bwd_kernel<D, TI><<<nb, 256, 0, st>>>(a); }
    { LaunchScope ls_("mixer_post_reduce", st); mixer_post_reduce_kernel<<<1, 256, 0, st>>>(a.dg_part, nb, D, dg); }
    return cudaGetLastError();
}

#define CYFA_DISPATCH_D(FN, ...)                                                       \
    switch (a.s.D) {                                                                   \
        case 64: return a.s.bf16 ? FN<64, __nv_bfloat16>(__VA_ARGS__) : FN<64, float>(__VA_ARGS__);    \
        case 128: return a.s.bf16 ? FN<128, __nv_bfloat16>(__VA_ARGS__) : FN<128, float>(__VA_ARGS__); \
        case 256: return a.s.bf16 ? FN<256, __nv_bfloat16>(__VA_ARGS__) : FN<256, float>(__VA_ARGS__); \
        default: return cudaErrorInvalidValue;                                         \
    }

}  // namespace

size_t mixer_workspace(const Shape& s) {
    const size_t pre = (size_t)3 * pre_splits(s, true) * s.B * s.H * s.D * KW * sizeof(float) +
                       (size_t)2 * pre_splits(s, true) * s.B * s.H * s.D * sizeof(float) + 256;
    const size_t post = (size_t)post_blocks(s) * s.D * sizeof(float);
    return pre > post ? pre : post;
}

cudaError_t launch_mixer_pre(const Shape& s, const void* const* x, const float* const* w,
                             const float* const* g, float eps, void* const* y, cudaStream_t st) {
    PreArgs a{};
    a.s = s;
    for (int z = 0; z < 3; ++z) {
        a.x[z] = x[z];
        a.w[z] = w[z];
        a.y[z] = y[z];
    }
    a.g[0] = g[0];
    a.g[1] = g[1];
    a.eps = eps;
    a.nsplit = pre_splits(s, false);
    float* const outs[5] = {nullptr, nullptr, nullptr, nullptr, nullptr};
    CYFA_DISPATCH_D(pre_launch, a, false, outs, st)
}

cudaError_t launch_mixer_pre_bwd(const Shape& s, const void* const* x, const float* const* w,
                                 const float* const* g, float eps, const void* const* dy,
                                 void* const* dx, float* const* dw, float* const* dg, void* ws,
                                 cudaStream_t st) {
    PreArgs a{};
    a.s = s;
    for (int z = 0; z < 3; ++z) {
        a.x[z] = x[z];
        a.w[z] = w[z];
        a.dy[z] = dy[z];
        a.dx[z] = dx[z];
    }
    a.g[0] = g[0];
    a.g[1] = g[1];
    a.eps = eps;
    a.nsplit = pre_splits(s, true);
    a.dw_part = static_cast<float*>(ws);
    a.dg_part = a.dw_part + (size_t)3 * a.nsplit * s.B * s.H * s.D * KW;
    float* const outs[5] = {dw[0], dw[1], dw[2], dg[0], dg[1]};
    CYFA_DISPATCH_D(pre_launch, a, true, outs, st)
}

cudaError_t launch_mixer_post(const Shape& s, const void* o, const void* z, const float* g,
                              float eps, void* y, cudaStream_t st) {
    PostArgs a{};
    a.s = s;
    a.o = o;
    a.zl = z;
    a.g = g;
    a.eps = eps;
    a.y = y;
    CYFA_DISPATCH_D(post_launch, a, false, nullptr, st)
}

cudaError_t launch_mixer_post_bwd(const Shape& s, const void* o, const void* z, const float* g,
                                  float eps, const void* dy, void* dO, void* dz, float* dg,
                                  void* ws, cudaStream_t st) {
    PostArgs a{};
    a.s = s;
    a.o = o;
    a.zl = z;
    a.g = g;
    a.eps = eps;
    a.dy = dy;
    a.dO = dO;
    a.dz = dz;
    a.dg_part = static_cast<float*>(ws);
    CYFA_DISPATCH_D(post_launch, a, true, dg, st)
}

}  // namespace cyfa
