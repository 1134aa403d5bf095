// Helpers shared by the tensor-core chunk kernels (forward and backward): 128-token chunks,
// the rotation-local Fourier row order, write vectors and rotations on half rows, TMEM half-row
// loads / stores, the thread roles of the 256-thread kernels.
#pragma once

#include <type_traits>

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

// The slot geometry a kernel instance works with: compile-time for m = 127, else the runtime
// values carried in the Shape.
template <class SL> __device__ __forceinline__ SL slots_of(const Shape& s);
// m = 127: every rotation pair is active and slot 127 alone is padding (no masks to evaluate)
template <class SL> __host__ __device__ constexpr bool full_slots() { return std::is_same<SL, Slots127>::value; }
template <> __device__ __forceinline__ Slots127 slots_of<Slots127>(const Shape&) { return {}; }
template <> __device__ __forceinline__ Slots slots_of<Slots>(const Shape& s) { return s.sl; }

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

// sin(pi x), cos(pi x) for a phase x in [0, 2) (a phase_pi value) on the special-function unit.
// The argument is first reduced to [-1, 1), where the unit's absolute error is about 2^-21: far
// below the fp16 rounding (2^-11 relative) of every tensor-core operand these angles feed.
__device__ __forceinline__ void sincospi_fast(float x, float* s, float* c) {
    if (x >= 1.f) x -= 2.f;
    __sincosf(3.14159265358979f * x, s, c);
}

// Rotation angles theta_j = 2 pi j lam / m for the 32 pairs of one column half, produced in
// order by angle addition from theta_1 (cos(x + y) = cos x cos y - sin x sin y,
// sin(x + y) = sin x cos y + cos x sin y), re-seeded from sincospi_fast every 16 steps.
template <class SL>
struct HalfAngles {
    float c1, s1, c, s, lam;
    int j0;
    SL sl;
    __device__ __forceinline__ HalfAngles(float lam_, int hf, const SL& sl_)
        : lam(lam_), j0(32 * hf + 1), sl(sl_) {
        sincospi_fast(phase_pi_m(lam, 1, sl), &s1, &c1);
        if (j0 == 1) {
            c = c1;
            s = s1;
        } else {
            sincospi_fast(phase_pi_m(lam, j0, sl), &s, &c);
        }
    }
    // advance to local pair jj (1..31)
    __device__ __forceinline__ void step(int jj) {
        if (jj == 16) {
            sincospi_fast(phase_pi_m(lam, j0 + 16, sl), &s, &c);
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
// Eq. app-b-explicit), in the tensor-core row order; the entries of pairs past (m-1)/2 are zero.
template <typename OT = __nv_bfloat16, class SL>
__device__ __forceinline__ void write_vector_half(uint8_t* tile, int r, int hf, float lam, float w,
                                                  const SL& sl) {
    float x[64];
    HalfAngles ang(lam, hf, sl);
    const float wa = w * sl.sqrt2_over_m;
#pragma unroll
    for (int jj = 0; jj < 32; ++jj) {
        if (jj > 0) ang.step(jj);
        const bool on = full_slots<SL>() || 32 * hf + jj + 1 <= sl.npair;
        x[jj] = on ? wa * ang.c : 0.f;
        x[jj + 32] = on ? -wa * ang.s : 0.f;
    }
    if (hf == 1) {
        x[31] = w * sl.inv_sqrt_m;
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

// ------------------------------------------------------------------ 512-thread column quarters
// In the 512-thread kernels warps w, w + 4, w + 8, w + 12 share TMEM lanes 32 (w % 4) .. + 31 and
// split a row's 128 columns into quarters cq = w / 4.  Quarter (hf, u) = (cq / 2, cq % 2) owns
// the 16 rotation pairs j = 32 hf + 16 u + i + 1 (i < 16) of the tensor-core order: element i
// of the thread's 32 values is column c0 + i (cosine entries) and element 16 + i is column
// c0 + 32 + i (sine entries), c0 = 64 hf + 16 u.  In quarter (1, 1) element 15 is the DC entry
// and element 31 the padding entry.
struct QRole {
    int warp, lane, q, cq, hf, u, row, c0;
    __device__ __forceinline__ QRole() {
        warp = threadIdx.x >> 5;
        lane = threadIdx.x & 31;
        q = warp & 3;
        cq = warp >> 2;
        hf = cq >> 1;
        u = cq & 1;
        row = 32 * q + lane;
        c0 = 64 * hf + 16 * u;
    }
};

// Angles of the 16 pairs of a quarter by angle addition from theta_1, seeded with sincospi_fast at
// the quarter's first pair (the same seeds as HalfAngles).
template <class SL>
struct QuarterAngles {
    float c1, s1, c, s;
    __device__ __forceinline__ QuarterAngles(float lam, int hf, int u, const SL& sl) {
        const int j0 = 32 * hf + 16 * u + 1;
        sincospi_fast(phase_pi_m(lam, 1, sl), &s1, &c1);
        if (j0 == 1) {
            c = c1;
            s = s1;
        } else {
            sincospi_fast(phase_pi_m(lam, j0, sl), &s, &c);
        }
    }
    __device__ __forceinline__ void step() {
        const float cn = c * c1 - s * s1;
        const float sn = s * c1 + c * s1;
        c = cn;
        s = sn;
    }
};

// The thread's 32 values <-> row r of a swizzled 16-bit tile (columns c0.. and c0 + 32..).
template <typename OT>
__device__ __forceinline__ void store_q(uint8_t* tile, int r, int c0, const float (&x)[32]) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float* v = x + 8 * k;
        uint4 w;
        w.x = pack2<OT>(v[0], v[1]);
        w.y = pack2<OT>(v[2], v[3]);
        w.z = pack2<OT>(v[4], v[5]);
        w.w = pack2<OT>(v[6], v[7]);
        *reinterpret_cast<uint4*>(tile + swz_off(r, c0 + 32 * (k >> 1) + 8 * (k & 1), 128)) = w;
    }
}
// fp16 tile -> fp32
__device__ __forceinline__ void load_q(const uint8_t* tile, int r, int c0, float (&x)[32]) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint4 w = *reinterpret_cast<const uint4*>(tile + swz_off(r, c0 + 32 * (k >> 1) + 8 * (k & 1), 128));
        const __half2* p = reinterpret_cast<const __half2*>(&w);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __half22float2(p[i]);
            x[8 * k + 2 * i] = f.x;
            x[8 * k + 2 * i + 1] = f.y;
        }
    }
}
// bf16 -> fp16 in place on the thread's 32 columns of row r
__device__ __forceinline__ void bf16_to_f16_q(uint8_t* tile, int r, int c0) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        uint4* p = reinterpret_cast<uint4*>(tile + swz_off(r, c0 + 32 * (k >> 1) + 8 * (k & 1), 128));
        uint4 w = *p;
        uint32_t* e = reinterpret_cast<uint32_t*>(&w);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&e[i]));
            e[i] = pack_f16(f.x, f.y);
        }
        *p = w;
    }
}
// multiply the thread's 32 columns of row r of an fp16 tile by w, in place
__device__ __forceinline__ void scale_q(uint8_t* tile, int r, int c0, float w) {
    float x[32];
    load_q(tile, r, c0, x);
#pragma unroll
    for (int i = 0; i < 32; ++i) x[i] *= w;
    store_q<__half>(tile, r, c0, x);
}

// 16 values (8 at column col, 8 at col + 32) -> row r of a swizzled 16-bit tile.
template <typename OT>
__device__ __forceinline__ void store8x2(uint8_t* tile, int r, int col, const float (&x)[16]) {
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const float* v = x + 8 * k;
        uint4 w;
        w.x = pack2<OT>(v[0], v[1]);
        w.y = pack2<OT>(v[2], v[3]);
        w.z = pack2<OT>(v[4], v[5]);
        w.w = pack2<OT>(v[6], v[7]);
        *reinterpret_cast<uint4*>(tile + swz_off(r, col + 32 * k, 128)) = w;
    }
}

// The quarter's entries of the write vector w U(-lam) b (Sec. 3.2), fp32; the entries of pairs
// past (m-1)/2 are zero.
template <class SL>
__device__ __forceinline__ void write_vector_q_vals(float (&x)[32], int hf, int u, float lam, float w,
                                                    const SL& sl) {
    QuarterAngles ang(lam, hf, u, sl);
    const float wa = w * sl.sqrt2_over_m;
    const int jb = 32 * hf + 16 * u + 1;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        if (i > 0) ang.step();
        const bool on = full_slots<SL>() || jb + i <= sl.npair;
        x[i] = on ? wa * ang.c : 0.f;
        x[16 + i] = on ? -wa * ang.s : 0.f;
    }
    if (hf == 1 && u == 1) {
        x[15] = w * sl.inv_sqrt_m;
        x[31] = 0.f;
    }
}
template <typename OT, class SL>
__device__ __forceinline__ void write_vector_q(uint8_t* tile, int r, int hf, int u, float lam, float w,
                                               const SL& sl) {
    float x[32];
    write_vector_q_vals(x, hf, u, lam, w, sl);
    store_q<OT>(tile, r, 64 * hf + 16 * u, x);
}

// x <- U(sign lam) x on the quarter's pairs; DC kept, padding zeroed.  (Pairs past (m-1)/2 hold
// zeros, which any rotation keeps.)
template <int SIGN, class SL>
__device__ __forceinline__ void rotate_q(float (&x)[32], int hf, int u, float lam, const SL& sl) {
    QuarterAngles ang(lam, hf, u, sl);
    const float dc = x[15];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        if (i > 0) ang.step();
        const float c = ang.c, sn = SIGN * ang.s;
        const float xc = x[i], xs = x[16 + i];
        x[i] = c * xc - sn * xs;
        x[16 + i] = sn * xc + c * xs;
    }
    if (hf == 1 && u == 1) {
        x[15] = dc;
        x[31] = 0.f;
    }
}

// <x, Omega y> over the quarter's pairs: sum_j (2 pi j / m) (x_sin,j y_cos,j - x_cos,j y_sin,j).
template <class SL>
__device__ __forceinline__ float omega_dot_q(const float (&x)[32], const float (&y)[32], int hf, int u,
                                             const SL& sl) {
    float acc = 0.f;
    const int jb = 32 * hf + 16 * u + 1;
    const float wb = sl.omega1 * (float)jb;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        if (jb + i <= sl.npair)
            acc += (wb + sl.omega1 * (float)i) * (x[16 + i] * y[i] - x[i] * y[16 + i]);
    }
    return acc;
}

// Softmax mask of the slot logits on the thread's 32 columns (element i is slot column
// c0 + (i & 15) + 32 (i >> 4)): true for the slots m..127 (padding), which leave the softmax.
template <class SL>
__device__ __forceinline__ bool slot_off(int c0, int i, const SL& sl) {
    if (full_slots<SL>()) return c0 == 64 + 16 && i == 31;   // slot 127 only
    return c0 + (i & 15) + 32 * (i >> 4) >= sl.m;
}

// x[i] = f x[i] + y[i] on 32 values, two per packed fp32 instruction (each lane rounds as fmaf).
__device__ __forceinline__ void fma2_scalar(float (&x)[32], float f, const float (&y)[32]) {
    const float2 f2 = make_float2(f, f);
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
        const float2 r = __ffma2_rn(f2, make_float2(x[i], x[i + 1]), make_float2(y[i], y[i + 1]));
        x[i] = r.x;
        x[i + 1] = r.y;
    }
}

// Causal decay mask on the thread's 32 columns (tokens t = c0 + 32 blk + i of this chunk) of
// row `row` (lane quarter q): x <- mul x 2^(g2 - g2_t) for t <= row, 0 otherwise, with g2 the
// row's log2-domain cumulative decay and s_g2[t] the column's.  Each 16-token block is classed
// for the whole warp (rows 32q .. 32q + 31), so no warp runs two paths:
//  * after every row of the warp: zero;
//  * before every row of the warp: 2^(g2 - g2_e) 2^(g2_e - g2_t), e the block's last token; both
//    factors are <= 1 (no overflow for any gate values), the first is one ex2 per thread and
//    block, the second (s_b[t] = 2^(s_g2[t | 15] - s_g2[t])) is shared by all rows;
//  * holding the diagonal of some row of the warp: one ex2 per entry.
// s_g2 and s_b are 16-byte aligned.  Every kernel pairing score matrices across the backward uses
// this with the same thread roles, so their score matrices agree bit for bit.
__device__ __forceinline__ void mask_decay_q(float (&x)[32], float mul, int row, int q, int c0,
                                             float g2, const float* s_g2, const float* s_b) {
#pragma unroll
    for (int blk = 0; blk < 2; ++blk) {
        const int tb = c0 + 32 * blk, te = tb + 15;
        float* xb = x + 16 * blk;
        if (tb >= 32 * (q + 1)) {
#pragma unroll
            for (int i = 0; i < 16; ++i) xb[i] = 0.f;
        } else if (te < 32 * q) {
            const float ar = mul * ex2(g2 - s_g2[te]);
            const float2 ar2 = make_float2(ar, ar);
            const float4* b4 = reinterpret_cast<const float4*>(s_b + tb);
#pragma unroll
            for (int k = 0; k < 4; ++k) {   // x *= ar * b, two lanes per packed instruction
                const float4 f = b4[k];
                const float2 lo = __fmul2_rn(make_float2(xb[4 * k], xb[4 * k + 1]),
                                             __fmul2_rn(ar2, make_float2(f.x, f.y)));
                const float2 hi = __fmul2_rn(make_float2(xb[4 * k + 2], xb[4 * k + 3]),
                                             __fmul2_rn(ar2, make_float2(f.z, f.w)));
                xb[4 * k + 0] = lo.x;
                xb[4 * k + 1] = lo.y;
                xb[4 * k + 2] = hi.x;
                xb[4 * k + 3] = hi.y;
            }
        } else {
            const float4* g4 = reinterpret_cast<const float4*>(s_g2 + tb);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float4 f = g4[k];
                const float gt[4] = {f.x, f.y, f.z, f.w};
#pragma unroll
                for (int m = 0; m < 4; ++m) {
                    const int t = tb + 4 * k + m;
                    const float e = ex2(g2 - gt[m]);
                    xb[4 * k + m] = (t <= row) ? mul * xb[4 * k + m] * e : 0.f;
                }
            }
        }
    }
}

// A [128][256] fp32 block staged in shared memory with rows padded to STAGE_LD floats (so that a
// warp's 16-byte stores to 32 different rows hit distinct banks) -> a contiguous global
// [128][256] block, every warp writing 512 contiguous bytes per instruction.  The caller has
// filled the stage and synchronised the block.
constexpr int STAGE_LD = 260;
__device__ __forceinline__ void stage_to_global_128x256(float* dst, const float* stage, int tid,
                                                        int nthreads) {
    for (int i = tid; i < 128 * 64; i += nthreads) {
        const int r = i >> 6, c4 = i & 63;
        *reinterpret_cast<float4*>(dst + r * 256 + 4 * c4) =
            *reinterpret_cast<const float4*>(stage + r * STAGE_LD + 4 * c4);
    }
}

__device__ __forceinline__ float dot32(const float (&x)[32], const float (&y)[32]) {
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < 32; ++i) acc = fmaf(x[i], y[i], acc);
    return acc;
}

}  // namespace
}  // namespace cyfa
