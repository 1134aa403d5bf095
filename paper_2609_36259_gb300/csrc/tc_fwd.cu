// Tensor-core (tcgen05 / TMEM / TMA) forward of the CyFA operator for bf16 inputs, d = 128.
//
// The chunk form of App. B (Eqs. app-cyfa-key-chunk and app-cyfa-value-chunk) is evaluated on
// 128-token chunks grouped into segments of SEGC chunks:
//   seg_state_tc : for every (b, h, segment), the segment's own contribution to the end-of-segment
//                  states, dS = A->^T [K | V] over all tokens of the segment, rows of A scaled by
//                  the decay from each token to the segment end (one TMEM accumulation);
//   seg_scan     : S_start(seg + 1) = exp(G_seg) S_start(seg) + dS(seg), elementwise in fp32;
//   seg_out_tc   : walks the segment's chunks with [Kbar | Vbar] resident in TMEM (fp32) and,
//                  per chunk, runs the eight products of the two passes and the middle readout
//                  (Sec. 3.3 Eq. cyfa-two-pass) on the tensor cores, then advances the state.
// States never round-trip through HBM at chunk granularity.  All operand tiles are 128 x 128 bf16
// in 128-byte-swizzled shared memory; accumulators are fp32 in TMEM.
#include "../../include/cyfa.h"
#include "common.cuh"
#include "kernels.h"
#include "tc_common.cuh"

namespace cyfa {

namespace {

using namespace tc;

constexpr int CT = 128;              // tokens per chunk on this path
constexpr int TILE = CT * 128 * 2;   // one 128 x 128 bf16 tile (32 KiB)
constexpr float LOG2E = 1.4426950408889634f;

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

// The 63 rotation angles theta_j = 2 pi j lam / m, produced in order by angle addition from
// theta_1 (cos(x + y) = cos x cos y - sin x sin y, sin(x + y) = sin x cos y + cos x sin y),
// re-seeded from sincospif every 16 steps to bound the rounding drift.
struct Angles {
    float c1, s1, c, s;
    float lam;
    __device__ __forceinline__ explicit Angles(float lam_) : lam(lam_) {
        sincospif(phase_pi(lam, 1), &s1, &c1);
        c = c1;
        s = s1;
    }
    // advance from pair j-1 to pair j (j >= 2)
    __device__ __forceinline__ void step(int j) {
        if (((j - 1) & 15) == 0) {
            sincospif(phase_pi(lam, j), &s, &c);
        } else {
            const float cn = c * c1 - s * s1;
            const float sn = s * c1 + c * s1;
            c = cn;
            s = sn;
        }
    }
};

// Store a 128-value fp32 row as bf16 into row r of a swizzled K-major tile.
__device__ __forceinline__ void store_row_bf16(uint8_t* tile, int r, const float (&x)[128]) {
#pragma unroll
    for (int q = 0; q < 16; ++q) {
        uint4 u;
        u.x = pack_bf16(x[8 * q + 0], x[8 * q + 1]);
        u.y = pack_bf16(x[8 * q + 2], x[8 * q + 3]);
        u.z = pack_bf16(x[8 * q + 4], x[8 * q + 5]);
        u.w = pack_bf16(x[8 * q + 6], x[8 * q + 7]);
        *reinterpret_cast<uint4*>(tile + swz_off(r, 8 * q, 128)) = u;
    }
}

// Temporal write vector w * U(-lam) b of one token (Sec. 3.2; b of Eq. app-b-explicit) as row r.
__device__ __forceinline__ void write_vector_row(uint8_t* tile, int r, float lam, float w) {
    float x[128];
    Angles ang(lam);
    const float wa = w * SQRT_2_OVER_M;
    x[0] = w * INV_SQRT_M;
#pragma unroll
    for (int j = 1; j <= NPAIR; ++j) {
        if (j > 1) ang.step(j);
        x[2 * j - 1] = wa * ang.c;
        x[2 * j] = -wa * ang.s;
    }
    x[127] = 0.f;
    store_row_bf16(tile, r, x);
}

// In-place x <- U(sign * lam) x on the pairs (2j-1, 2j); the DC entry is untouched and the
// padding entry set to 0.
template <int SIGN>
__device__ __forceinline__ void rotate_row(float (&x)[128], float lam) {
    Angles ang(lam);
#pragma unroll
    for (int j = 1; j <= NPAIR; ++j) {
        if (j > 1) ang.step(j);
        const float c = ang.c, s = SIGN * ang.s;
        const float xc = x[2 * j - 1], xs = x[2 * j];
        x[2 * j - 1] = c * xc - s * xs;
        x[2 * j] = s * xc + c * xs;
    }
    x[127] = 0.f;
}

__device__ __forceinline__ void tmem_ld_row(uint32_t taddr, float (&x)[128]) {
    float v[32];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        tmem_ld32(taddr + 32 * q, v);
#pragma unroll
        for (int i = 0; i < 32; ++i) x[32 * q + i] = v[i];
    }
}

// ---------------------------------------------------------------------------------------
template <int SEGC>
__global__ void __launch_bounds__(128) seg_state_tc(const __grid_constant__ CUtensorMap tk,
                                                     const __grid_constant__ CUtensorMap tv,
                                                     TcFwdArgs a) {
    const Shape s = a.s;
    const int seg = blockIdx.x, bh = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nct = s.T / CT;
    const int c_begin = seg * SEGC;
    const int nc = min(SEGC, nct - c_begin);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    // [buf][A | K | V] tiles
    uint8_t* tiles = smem;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 6 * TILE);   // tma[2], mma[2]
    uint32_t* s_taddr = reinterpret_cast<uint32_t*>(bars + 4);
    float* s_tot = reinterpret_cast<float*>(s_taddr + 4);            // [SEGC]
    float* s_sfx = s_tot + SEGC;                                     // [SEGC]

    if (tid == 0) {
        for (int i = 0; i < 4; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    if (warp == 0) tmem_alloc(s_taddr, 256);
    if (tid < nc) {
        const int t0 = (c_begin + tid) * CT;
        s_tot[tid] = cum128(s, a.g, b, h, t0, t0 + CT - 1);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *s_taddr;
    if (tid == 0) {
        float acc = 0.f;
        for (int c = nc - 1; c >= 0; --c) {
            s_sfx[c] = acc;
            acc += s_tot[c];
        }
        a.segG[(size_t)bh * a.nseg + seg] = acc;
    }
    auto issue_kv = [&](int c, int buf) {
        uint8_t* tK = tiles + (3 * buf + 1) * TILE;
        uint8_t* tV = tiles + (3 * buf + 2) * TILE;
        const int row = b * s.T + (c_begin + c) * CT;
        mbar_expect_tx(&bars[buf], 2 * TILE);
        tma_load_3d(tK, &tk, 0, h, row, &bars[buf]);
        tma_load_3d(tK + TILE / 2, &tk, 64, h, row, &bars[buf]);
        tma_load_3d(tV, &tv, 0, h, row, &bars[buf]);
        tma_load_3d(tV + TILE / 2, &tv, 64, h, row, &bars[buf]);
    };
    if (tid == 0) issue_kv(0, 0);
    __syncthreads();
    bool ok = true;
    const uint32_t idesc = idesc_bf16(128, 128, 1, 1);
    for (int c = 0; c < nc; ++c) {
        const int buf = c & 1;
        if (c >= 1 && ok) ok = mbar_wait(&bars[2 + ((c - 1) & 1)], ((c - 1) >> 1) & 1);
        if (tid == 0 && ok && c + 1 < nc) issue_kv(c + 1, (c + 1) & 1);
        // A-> rows of this chunk, scaled by the decay from the token to the segment end
        {
            const int t0 = (c_begin + c) * CT, t = t0 + tid;
            const size_t gi = ((size_t)b * s.T + t) * s.H + h;
            const float w = a.beta[gi] *
                            ex2((s_tot[c] - cum128(s, a.g, b, h, t0, t) + s_sfx[c]) * LOG2E);
            write_vector_row(tiles + 3 * buf * TILE, tid, a.lam[gi], w);
        }
        fence_async_smem();
        ok = __syncthreads_and(ok);
        if (!ok) break;
        if (tid == 0) {
            if (mbar_wait(&bars[buf], (c >> 1) & 1)) {
                tc_fence_after();
                const uint32_t tA = smem_u32(tiles + 3 * buf * TILE);
                const uint32_t tK = smem_u32(tiles + (3 * buf + 1) * TILE);
                const uint32_t tV = smem_u32(tiles + (3 * buf + 2) * TILE);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    mma_bf16(taddr, mnmajor_desc(tA, 128, k), mnmajor_desc(tK, 128, k), idesc,
                             (c > 0 || k > 0) ? 1u : 0u);
                    mma_bf16(taddr + 128, mnmajor_desc(tA, 128, k), mnmajor_desc(tV, 128, k),
                             idesc, (c > 0 || k > 0) ? 1u : 0u);
                }
                mma_commit(&bars[2 + buf]);
            }
        }
    }
    if (ok) ok = mbar_wait(&bars[2 + ((nc - 1) & 1)], ((nc - 1) >> 1) & 1);
    tc_fence_after();
    ok = __syncthreads_and(ok);
    if (ok) {
        const int row = warp * 32 + lane;
        float* dst = a.segS + (((size_t)bh * a.nseg + seg) * 128 + row) * 256;
        for (int c0 = 0; c0 < 256; c0 += 32) {
            float v[32];
            tmem_ld32(taddr + ((uint32_t)(warp * 32) << 16) + c0, v);
#pragma unroll
            for (int i = 0; i < 32; i += 4)
                *reinterpret_cast<float4*>(dst + c0 + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
        }
    } else if (tid == 0) {
        flag_error(CYFA_ERR_TIMEOUT);
        // let copies still in flight land before the shared memory is released
        for (int i = 0; i < 2; ++i) mbar_wait(&bars[i], 0);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(taddr, 256);
}

// Segment-start states: S_start(0) = initial state, S_start(j+1) = exp(G_j) S_start(j) + dS(j),
// in place over the dS buffer; the final state goes to Kout / Vout (paper row order).
__global__ void __launch_bounds__(256) seg_scan_kernel(TcFwdArgs a) {
    const int bh = blockIdx.y;
    const int e = blockIdx.x * 256 + threadIdx.x;   // element of the [128 x 256] state block
    const int row = e >> 8, col = e & 255;
    const bool isK = col < 128;
    const int dcol = col & 127;
    float S = 0.f;
    const float* init = isK ? a.Kbar0 : a.Vbar0;
    if (init) S = init[((size_t)bh * 128 + row) * 128 + dcol];
    for (int j = 0; j < a.nseg; ++j) {
        float* p = a.segS + ((size_t)bh * a.nseg + j) * 128 * 256 + e;
        const float dS = *p;
        *p = S;
        S = expf(a.segG[(size_t)bh * a.nseg + j]) * S + dS;
    }
    float* out = isK ? a.Kout : a.Vout;
    if (out) out[((size_t)bh * 128 + row) * 128 + dcol] = S;
}

// ---------------------------------------------------------------------------------------
template <int SEGC>
__global__ void __launch_bounds__(128) seg_out_tc(const __grid_constant__ CUtensorMap tq,
                                                   const __grid_constant__ CUtensorMap tk,
                                                   const __grid_constant__ CUtensorMap tv,
                                                   const __grid_constant__ CUtensorMap tm,
                                                   TcFwdArgs a) {
    const Shape s = a.s;
    const int seg = blockIdx.x, bh = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nct = s.T / CT;
    const int c_begin = seg * SEGC;
    const int nc = min(SEGC, nct - c_begin);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    uint8_t* T_Q = smem;               // Q, later A-> (state-update operand)
    uint8_t* T_K = smem + 1 * TILE;
    uint8_t* T_V = smem + 2 * TILE;
    uint8_t* T_A = smem + 3 * TILE;    // write vectors a_s (rows = tokens)
    uint8_t* T_S = smem + 4 * TILE;    // staging: P1, z, p, O'', P2 (rows = tokens)
    uint8_t* T_N = smem + 5 * TILE;    // state snapshot: Kbar, then Vbar (rows = slots)
    uint8_t* T_M = smem + 6 * TILE;    // M = R Phi (rows = slots r, cols = Fourier index)
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 7 * TILE);   // tma, mma, m
    uint32_t* s_taddr = reinterpret_cast<uint32_t*>(bars + 4);
    float* s_g2 = reinterpret_cast<float*>(s_taddr + 4);             // [128] log2-domain decays

    if (tid == 0) {
        for (int i = 0; i < 3; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    if (warp == 0) tmem_alloc(s_taddr, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *s_taddr;
    const uint32_t tl = taddr + ((uint32_t)(warp * 32) << 16);   // this warp's lane quarter
    const uint32_t S_COL = 0, X1 = 256, X2 = 384;

    auto issue_qkv = [&](int c) {
        const int row = b * s.T + (c_begin + c) * CT;
        mbar_expect_tx(&bars[0], 3 * TILE);
        tma_load_3d(T_Q, &tq, 0, h, row, &bars[0]);
        tma_load_3d(T_Q + TILE / 2, &tq, 64, h, row, &bars[0]);
        tma_load_3d(T_K, &tk, 0, h, row, &bars[0]);
        tma_load_3d(T_K + TILE / 2, &tk, 64, h, row, &bars[0]);
        tma_load_3d(T_V, &tv, 0, h, row, &bars[0]);
        tma_load_3d(T_V + TILE / 2, &tv, 64, h, row, &bars[0]);
    };
    if (tid == 0) {
        mbar_expect_tx(&bars[2], TILE);
        tma_load_2d(T_M, &tm, 0, h * 128, &bars[2]);
        tma_load_2d(T_M + TILE / 2, &tm, 64, h * 128, &bars[2]);
        issue_qkv(0);
    }
    // segment-start state into TMEM, Kbar snapshot into T_N (row = slot = tid)
    {
        const float* src = a.segS + (((size_t)bh * a.nseg + seg) * 128 + tid) * 256;
        float kr[128];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            float v[32];
#pragma unroll
            for (int i = 0; i < 32; i += 4) {
                const float4 f = *reinterpret_cast<const float4*>(src + 32 * q + i);
                v[i] = f.x; v[i + 1] = f.y; v[i + 2] = f.z; v[i + 3] = f.w;
            }
            tmem_st32(tl + S_COL + 32 * q, v);
            if (q < 4) {
#pragma unroll
                for (int i = 0; i < 32; ++i) kr[32 * q + i] = v[i];
            }
        }
        store_row_bf16(T_N, tid, kr);
    }
    fence_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    bool ok = mbar_wait(&bars[2], 0);
    ok = __syncthreads_and(ok);
    uint32_t tma_ph = 0, mma_ph = 0;
    const float scale = s.scale;
    const uint32_t id_kk = idesc_bf16(128, 128, 0, 0);
    const uint32_t id_kn = idesc_bf16(128, 128, 0, 1);
    const uint32_t id_nn = idesc_bf16(128, 128, 1, 1);
    const uint32_t uQ = smem_u32(T_Q), uK = smem_u32(T_K), uV = smem_u32(T_V),
                   uA = smem_u32(T_A), uS = smem_u32(T_S), uN = smem_u32(T_N),
                   uM = smem_u32(T_M);

    // all threads: wait for the MMAs committed so far, then order TMEM reads after them
    auto wait_mma = [&]() {
        if (ok) ok = mbar_wait(&bars[1], mma_ph);
        mma_ph ^= 1;
        tc_fence_after();
    };
    auto mma_ok = [&]() { return tid == 0 && ok; };
    // all threads: publish shared-memory operand writes (and TMEM stores) to the MMA thread
    // (the block agrees on `ok`, so every later branch on it is uniform)
    auto publish = [&]() {
        fence_async_smem();
        tc_fence_before();
        ok = __syncthreads_and(ok);
        tc_fence_after();
    };

    for (int c = 0; c < nc && ok; ++c) {
        const int t0 = (c_begin + c) * CT;
        const int tok = t0 + tid;
        const size_t gi = ((size_t)b * s.T + tok) * s.H + h;
        const float lam = a.lam[gi];
        const float beta = a.beta[gi];
        const float g2 = cum128(s, a.g, b, h, t0, tok) * LOG2E;
        s_g2[tid] = g2;
        write_vector_row(T_A, tid, lam, beta);
        publish();
        if (!ok) break;
        const float g2C = s_g2[CT - 1];
        const float gam = ex2(g2);

        // X1 = Q K^T, X2 = Q Kbar^T
        if (mma_ok()) {
            ok = mbar_wait(&bars[0], tma_ph);
            if (ok) {
                tc_fence_after();
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    mma_bf16(taddr + X1, kmajor_desc(uQ, 128, k), kmajor_desc(uK, 128, k), id_kk, k > 0);
                    mma_bf16(taddr + X2, kmajor_desc(uQ, 128, k), kmajor_desc(uN, 128, k), id_kk, k > 0);
                }
                mma_commit(&bars[1]);
            }
        }
        tma_ph ^= 1;
        wait_mma();
        // P1 = s (Q K^T) o Gamma
        {
            float x[128];
            tmem_ld_row(tl + X1, x);
#pragma unroll
            for (int j = 0; j < 128; ++j)
                x[j] = (j <= tid) ? scale * x[j] * ex2(g2 - s_g2[j]) : 0.f;
            store_row_bf16(T_S, tid, x);
        }
        publish();
        if (!ok) break;
        if (mma_ok()) {
#pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X1, kmajor_desc(uS, 128, k), mnmajor_desc(uA, 128, k), id_kn, k > 0);
            mma_commit(&bars[1]);
        }
        // A-> rows into T_Q (Q is consumed), Vbar snapshot into T_N, state scaled by gamma^C
        write_vector_row(T_Q, tid, lam, beta * ex2(g2C - g2));
        {
            const float gC = ex2(g2C);
            float vr[128];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                float v[32];
                tmem_ld32(tl + S_COL + 32 * q, v);
                if (q >= 4) {
#pragma unroll
                    for (int i = 0; i < 32; ++i) vr[32 * (q - 4) + i] = v[i];
                }
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] *= gC;
                tmem_st32(tl + S_COL + 32 * q, v);
            }
            store_row_bf16(T_N, tid, vr);
        }
        publish();
        if (!ok) break;
        if (mma_ok()) {
            // state update: [Kbar | Vbar] += A->^T [K | V]
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                mma_bf16(taddr + S_COL, mnmajor_desc(uQ, 128, k), mnmajor_desc(uK, 128, k), id_nn, 1u);
                mma_bf16(taddr + S_COL + 128, mnmajor_desc(uQ, 128, k), mnmajor_desc(uV, 128, k), id_nn, 1u);
            }
        }
        wait_mma();   // P1 A
        // z = U(lam) o',  o' = s gamma_r (Q Kbar^T) + P1 A
        {
            float x[128], y[32];
            tmem_ld_row(tl + X2, x);
            const float f = scale * gam;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                tmem_ld32(tl + X1 + 32 * q, y);
#pragma unroll
                for (int i = 0; i < 32; ++i) x[32 * q + i] = fmaf(f, x[32 * q + i], y[i]);
            }
            rotate_row<1>(x, lam);
            store_row_bf16(T_S, tid, x);
        }
        publish();
        if (!ok) break;
        if (mma_ok()) {
#pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X1, kmajor_desc(uS, 128, k), kmajor_desc(uM, 128, k), id_kk, k > 0);
            mma_commit(&bars[1]);
        }
        wait_mma();   // also covers the state update issued before this commit
        // p = softmax over the 127 active slots of l = z M^T
        {
            float x[128];
            tmem_ld_row(tl + X1, x);
            float mx = -INFINITY;
#pragma unroll
            for (int j = 0; j < MA; ++j) mx = fmaxf(mx, x[j]);
            float sum = 0.f;
#pragma unroll
            for (int j = 0; j < MA; ++j) {
                x[j] = ex2((x[j] - mx) * LOG2E);
                sum += x[j];
            }
            const float inv = 1.f / sum;
#pragma unroll
            for (int j = 0; j < MA; ++j) x[j] *= inv;
            x[127] = 0.f;
            store_row_bf16(T_S, tid, x);
        }
        publish();
        if (!ok) break;
        if (mma_ok()) {
#pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X2, kmajor_desc(uS, 128, k), mnmajor_desc(uM, 128, k), id_kn, k > 0);
            mma_commit(&bars[1]);
        }
        wait_mma();
        // o'' = U(-lam) (p M)
        {
            float x[128];
            tmem_ld_row(tl + X2, x);
            rotate_row<-1>(x, lam);
            store_row_bf16(T_S, tid, x);
        }
        publish();
        if (!ok) break;
        if (mma_ok()) {
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                mma_bf16(taddr + X1, kmajor_desc(uS, 128, k), kmajor_desc(uA, 128, k), id_kk, k > 0);
                mma_bf16(taddr + X2, kmajor_desc(uS, 128, k), mnmajor_desc(uN, 128, k), id_kn, k > 0);
            }
            mma_commit(&bars[1]);
        }
        wait_mma();
        // P2 = (O'' A^T) o Gamma
        {
            float x[128];
            tmem_ld_row(tl + X1, x);
#pragma unroll
            for (int j = 0; j < 128; ++j) x[j] = (j <= tid) ? x[j] * ex2(g2 - s_g2[j]) : 0.f;
            store_row_bf16(T_S, tid, x);
        }
        publish();
        if (!ok) break;
        if (mma_ok()) {
#pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X1, kmajor_desc(uS, 128, k), mnmajor_desc(uV, 128, k), id_kn, k > 0);
            mma_commit(&bars[1]);
        }
        wait_mma();
        // next chunk's tiles (Q, K, V are consumed), then o = gamma_r (O'' Vbar) + P2 V
        if (mma_ok() && c + 1 < nc) issue_qkv(c + 1);
        {
            float x[128], y[32];
            tmem_ld_row(tl + X2, x);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                tmem_ld32(tl + X1 + 32 * q, y);
#pragma unroll
                for (int i = 0; i < 32; ++i) x[32 * q + i] = fmaf(gam, x[32 * q + i], y[i]);
            }
            __nv_bfloat16* O = static_cast<__nv_bfloat16*>(a.o) + gi * 128;
#pragma unroll
            for (int q = 0; q < 16; ++q) {
                uint4 u;
                u.x = pack_bf16(x[8 * q + 0], x[8 * q + 1]);
                u.y = pack_bf16(x[8 * q + 2], x[8 * q + 3]);
                u.z = pack_bf16(x[8 * q + 4], x[8 * q + 5]);
                u.w = pack_bf16(x[8 * q + 6], x[8 * q + 7]);
                *reinterpret_cast<uint4*>(O + 8 * q) = u;
            }
        }
        // Kbar snapshot of the next chunk's start state
        {
            float kr[128];
            tmem_ld_row(tl + S_COL, kr);
            store_row_bf16(T_N, tid, kr);
        }
        publish();
    }
    if (!ok && lane == 0) flag_error(CYFA_ERR_TIMEOUT);
    // let copies still in flight land before the shared memory is released
    if (!ok && tid == 0) {
        mbar_wait(&bars[0], tma_ph);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(taddr, 512);
}

__global__ void m_to_bf16_kernel(const float* M, __nv_bfloat16* Mb, int n) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) Mb[i] = __float2bfloat16_rn(M[i]);
}

constexpr int SEGC_DEFAULT = 8;    // 1024-token segments

}  // namespace

int tc_fwd_segments(const Shape& s) {
    const int nct = s.T / CT;
    return (nct + SEGC_DEFAULT - 1) / SEGC_DEFAULT;
}

bool tc_fwd_supported(const Shape& s) { return s.bf16 && s.D == 128 && s.T % CT == 0; }

cudaError_t launch_fwd_tc(const TcFwdArgs& a, const void* q, const void* k, const void* v,
                          const float* Mf, cudaStream_t st) {
    const Shape& s = a.s;
    CUtensorMap mq, mk, mv, mm;
    const unsigned long long dims[3] = {128ull, (unsigned long long)s.H,
                                        (unsigned long long)s.B * s.T};
    const unsigned long long strides[2] = {128ull * 2, (unsigned long long)s.H * 128 * 2};
    const unsigned box[3] = {64, 1, CT};
    const unsigned long long mdims[2] = {128ull, (unsigned long long)s.H * 128};
    const unsigned long long mstr[1] = {256ull};
    const unsigned mbox[2] = {64, 128};
    if (!make_tmap_bf16(&mq, q, 3, dims, strides, box) || !make_tmap_bf16(&mk, k, 3, dims, strides, box) ||
        !make_tmap_bf16(&mv, v, 3, dims, strides, box) ||
        !make_tmap_bf16(&mm, a.Mb, 2, mdims, mstr, mbox))
        return cudaErrorInvalidValue;
    const int n = s.H * 128 * 128;
    {
        LaunchScope ls_("m_to_bf16", st);
        m_to_bf16_kernel<<<(n + 255) / 256, 256, 0, st>>>(Mf, const_cast<__nv_bfloat16*>(a.Mb), n);
    }
    const dim3 grid(a.nseg, s.B * s.H);
    const int smA = 6 * TILE + 1024 + 256;
    auto kA = seg_state_tc<SEGC_DEFAULT>;
    cudaFuncSetAttribute(kA, cudaFuncAttributeMaxDynamicSharedMemorySize, smA);
    { LaunchScope ls_("tc_seg_state", st); kA<<<grid, 128, smA, st>>>(mk, mv, a); }
    { LaunchScope ls_("tc_seg_scan", st); seg_scan_kernel<<<dim3(128, s.B * s.H), 256, 0, st>>>(a); }
    const int smC = 7 * TILE + 1024 + 1024;
    auto kC = seg_out_tc<SEGC_DEFAULT>;
    cudaFuncSetAttribute(kC, cudaFuncAttributeMaxDynamicSharedMemorySize, smC);
    { LaunchScope ls_("tc_seg_out", st); kC<<<grid, 128, smC, st>>>(mq, mk, mv, mm, a); }
    return cudaGetLastError();
}

cudaError_t tc_read_error(cudaStream_t st, int* err) {
    cudaError_t e = cudaMemcpyFromSymbolAsync(err, g_tc_err, sizeof(int), 0,
                                              cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return e;
    e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return e;
    if (*err) {
        int zero = 0;
        e = cudaMemcpyToSymbol(g_tc_err, &zero, sizeof(int));
    }
    return e;
}

}  // namespace cyfa
