// Helpers shared by the tensor-core chunk kernels (forward and backward): 128-token chunks,
// the rotation-local Fourier row order, write vectors and rotations on half rows, TMEM half-row
// loads / stores, the thread roles of the 256-thread kernels.
#pragma once

#include "../../include/cyfa.h"
#include "common.cuh"
#include "kernels.h"
#include "tc_common.cuh"

namespace cyfa {
namespace {

using namespace tc;

constexpr int CT = 128;              // tokens per chunk on this path
constexpr int TC_SEGC = 8;           // chunks per segment (1024 tokens)
constexpr int TILE = CT * 128 * 2;   // one 128 x 128 bf16 tile (32 KiB)
constexpr float LOG2E = 1.4426950408889634f;

// error word of the including translation unit (each has its own copy)
static __device__ int g_tc_err;

__device__ __forceinline__ void flag_error(int code) { atomicExch(&g_tc_err, code); }

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// g_cum of token t rebased to the start of its 128-token chunk t0 (g_cum is local to s.Cg).
__device__ __forceinline__ float cum128(const Shape& s, const float* g, int b, int h, int t0,
                                       int t) {
    float v = g[((size_t)b * s.T + t) * s.H + h];
    if (s.Cg == 64 && t - t0 >= 64) v += g[((size_t)b * s.T + t0 + 63) * s.H + h];
    return v;
}

// Order of the 128 Fourier-axis rows inside the tensor-core kernels.  Column half hf (0 or 1)
// holds the pairs j = 32 hf + jj + 1 (jj < 32): cosine entry at 64 hf + jj, sine entry at
// 64 hf + jj + 32, so every rotation block of U lies inside one half.  The DC entry sits at 95
// and the padding entry at 127.  Exported / imported states use the paper's order
// [DC, cos_1, sin_1, ..., cos_63, sin_63, pad]; these map between the two.
__host__ __device__ __forceinline__ int tc_slot(int p) {
    if (p == 0) return 95;
    if (p == 127) return 127;
    const int j = (p + 1) >> 1, hf = (j - 1) >> 5, jj = (j - 1) & 31;
    return 64 * hf + jj + ((p & 1) ? 0 : 32);
}
__host__ __device__ __forceinline__ int paper_slot(int t) {
    if (t == 95) return 0;
    if (t == 127) return 127;
    const int hf = t >> 6, l = t & 63, jj = l & 31;
    const int j = 32 * hf + jj + 1;
    return (l >= 32) ? 2 * j : 2 * j - 1;
}

// Rotation angles theta_j = 2 pi j lam / m for the 32 pairs of one column half, produced in
// order by angle addition from theta_1 (cos(x + y) = cos x cos y - sin x sin y,
// sin(x + y) = sin x cos y + cos x sin y), re-seeded from sincospif every 16 steps.
struct HalfAngles {
    float c1, s1, c, s, lam;
    int j0;
    __device__ __forceinline__ HalfAngles(float lam_, int hf) : lam(lam_), j0(32 * hf + 1) {
        sincospif(phase_pi(lam, 1), &s1, &c1);
        if (j0 == 1) {
            c = c1;
            s = s1;
        } else {
            sincospif(phase_pi(lam, j0), &s, &c);
        }
    }
    // advance to local pair jj (1..31)
    __device__ __forceinline__ void step(int jj) {
        if (jj == 16) {
            sincospif(phase_pi(lam, j0 + 16), &s, &c);
        } else {
            const float cn = c * c1 - s * s1;
            const float sn = s * c1 + c * s1;
            c = cn;
            s = sn;
        }
    }
};

// Store 64 fp32 values as 16-bit OT into columns [64 hf, 64 hf + 64) of row r of a swizzled tile.
template <typename OT = __nv_bfloat16>
__device__ __forceinline__ void store_half_bf16(uint8_t* tile, int r, int hf, const float (&x)[64]) {
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        uint4 u;
        u.x = pack2<OT>(x[8 * q + 0], x[8 * q + 1]);
        u.y = pack2<OT>(x[8 * q + 2], x[8 * q + 3]);
        u.z = pack2<OT>(x[8 * q + 4], x[8 * q + 5]);
        u.w = pack2<OT>(x[8 * q + 6], x[8 * q + 7]);
        *reinterpret_cast<uint4*>(tile + swz_off(r, 64 * hf + 8 * q, 128)) = u;
    }
}

// One column half of the temporal write vector w U(-lam) b of a token (Sec. 3.2, b of
// Eq. app-b-explicit), in the tensor-core row order.
template <typename OT = __nv_bfloat16>
__device__ __forceinline__ void write_vector_half(uint8_t* tile, int r, int hf, float lam, float w) {
    float x[64];
    HalfAngles ang(lam, hf);
    const float wa = w * SQRT_2_OVER_M;
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
        if (jj > 0) ang.step(jj);
        x[jj] = wa * ang.c;
        x[jj + 32] = -wa * ang.s;
    }
    if (hf == 1) {
        x[31] = w * INV_SQRT_M;
        x[63] = 0.f;
    }
    store_half_bf16<OT>(tile, r, hf, x);
}

// Convert columns [64 hf, +64) of row r of a swizzled tile from bf16 to fp16 in place (exact
// for every value in fp16's normal range; the TMA loads the bf16 inputs as they are).
__device__ __forceinline__ void bf16_to_f16_half(uint8_t* tile, int r, int hf) {
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        uint4* p = reinterpret_cast<uint4*>(tile + swz_off(r, 64 * hf + 8 * q, 128));
        uint4 u = *p;
        uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[i]));
            w[i] = pack_f16(f.x, f.y);
        }
        *p = u;
    }
}

// x <- U(sign lam) x on one column half (tensor-core row order); DC kept, padding zeroed.
template <int SIGN>
__device__ __forceinline__ void rotate_half(float (&x)[64], int hf, float lam) {
    HalfAngles ang(lam, hf);
    const float dc = x[31];
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
        if (jj > 0) ang.step(jj);
        const float c = ang.c, s = SIGN * ang.s;
        const float xc = x[jj], xs = x[jj + 32];
        x[jj] = c * xc - s * xs;
        x[jj + 32] = s * xc + c * xs;
    }
    if (hf == 1) {
        x[31] = dc;
        x[63] = 0.f;
    }
}

__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float (&x)[64]) {
    float v[32];
    tmem_ld32(taddr, v);
#pragma unroll
    for (int i = 0; i < 32; ++i) x[i] = v[i];
    tmem_ld32(taddr + 32, v);
#pragma unroll
    for (int i = 0; i < 32; ++i) x[32 + i] = v[i];
}
__device__ __forceinline__ void tmem_st64(uint32_t taddr, const float (&x)[64]) {
    float v[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = x[i];
    tmem_st32(taddr, v);
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = x[32 + i];
    tmem_st32(taddr + 32, v);
}

// Lane quarter / column half owned by this thread in the 256-thread tensor-core kernels:
// warps w and w + 4 share TMEM lanes 32 (w % 4) .. + 31 (one row each per thread) and split the
// 128 columns of a tile into halves hf = w / 4.
struct Role {
    int warp, lane, q, hf, row;
    __device__ __forceinline__ Role() {
        warp = threadIdx.x >> 5;
        lane = threadIdx.x & 31;
        q = warp & 3;
        hf = warp >> 2;
        row = 32 * q + lane;
    }
};

}  // namespace
}  // namespace cyfa
