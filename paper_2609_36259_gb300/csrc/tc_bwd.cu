// Tensor-core (tcgen05 / TMEM / TMA) backward of the CyFA operator for bf16 inputs, d = 128.
// Every tensor-core operand of the backward is fp16: the bf16 inputs are converted exactly in
// shared memory after their TMA loads, and the stored intermediates (states, adjoints, o'', dO',
// score matrices) carry fp16's 11-bit significand.  The clock gradient is a difference of
// nearly cancelling paths (<dz, Omega z> against <do'', Omega o''>), so the 8-bit significand of
// bf16 intermediates would show in it at long sequence lengths.
//
// Gradient of sum(o * dO) through the chunk form of App. B and the middle line of Sec. 3.3
// Eq. cyfa-two-pass, on 128-token chunks (segments of TC_SEGC chunks):
//   forward segment states (tc_fwd.cu)  S_start per segment;
//   snap_fwd_tc   walks each segment and stores the fp16 chunk-start states [Kbar | Vbar];
//   bwd_chunk1_tc per chunk: recompute O', O''; dO'' = gamma (dO Vbar^T) + (dO V^T o Gamma) A;
//                 the middle readout's gradient (softmax backward through R Phi) gives dO';
//                 dq = s [gamma (dO' Kbar) + (dO' A^T o Gamma) K]; stores o'', dO' and the
//                 per-token scalars <o'', do''> + <q~, dq~> and <dz, Omega z> - <do'', Omega o''>;
//   adj_walk_tc   the adjoint states of the reversed recurrence
//                 D_c = gamma^C D_{c+1} + sum_r gamma^r [dO'_r q~_r^T | o''_r dO_r^T]:
//                 per-segment contributions, a reverse segment scan, then per-chunk snapshots;
//   bwd_chunk2_tc per chunk: dK = P3^T Q~ + A-> D^K, dV = P2^T dO + A-> D^V,
//                 dA = P4^T O'' + V-> D^V^T + P1^T dO' + K-> D^K^T (rows -> scaled by
//                 gamma^C / gamma^s), and the per-token scalars of the gate gradients;
//   tc_gate       the reverse cumulative sums of App. D.1 (d delta_s = sum_{t>=s} d lambda_t,
//                 d log alpha_s = sum_{t>=s} dG_t), split at the end of s's chunk: the tokens of
//                 the chunk are summed directly, everything after the chunk enters as one
//                 state-level term.  Moving the clock of every later token by e is, by the
//                 clock-origin invariance of Prop. 6, the same as rotating the chunk-end states
//                 S by U(e); raising the log-decay of every later token by e is the same as
//                 scaling S by exp(e).  So the later tokens contribute <D, Omega S> to the clock
//                 gradient and <D, S> to the decay gradient, with D the adjoint of S.  This keeps
//                 the per-token terms, which are small differences of large products, from being
//                 summed over the whole sequence.
#include "tc_chunk.cuh"

namespace cyfa {

namespace {

using namespace tc;

__device__ __forceinline__ void load_gates_row(const Shape& s, const TcBwdArgs& a, int b, int h,
                                               int t0, int row, float& lam, float& beta,
                                               float& g) {
    const size_t gi = ((size_t)b * s.T + t0 + row) * s.H + h;
    lam = a.lam[gi];
    beta = a.beta[gi];
    g = cum128(s, a.g, b, h, t0, t0 + row);
}

// 64 fp32 values -> 16-bit OT at dst (plain row-major, 128 bytes)
template <typename OT>
__device__ __forceinline__ void store_global_half(OT* dst, const float (&x)[64]) {
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        uint4 u;
        u.x = pack2<OT>(x[8 * q + 0], x[8 * q + 1]);
        u.y = pack2<OT>(x[8 * q + 2], x[8 * q + 3]);
        u.z = pack2<OT>(x[8 * q + 4], x[8 * q + 5]);
        u.w = pack2<OT>(x[8 * q + 6], x[8 * q + 7]);
        *reinterpret_cast<uint4*>(dst + 8 * q) = u;
    }
}

// eight fp16 values -> fp32
__device__ __forceinline__ void unpack8(const uint4& u, float* f) {
    const __half2* p = reinterpret_cast<const __half2*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 t = __half22float2(p[i]);
        f[2 * i] = t.x;
        f[2 * i + 1] = t.y;
    }
}

// Columns [64 hf, 64 hf + 64) of row r of a swizzled fp16 tile, as fp32.
__device__ __forceinline__ void load_half_smem(const uint8_t* tile, int r, int hf, float (&x)[64]) {
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        const uint4 u = *reinterpret_cast<const uint4*>(tile + swz_off(r, 64 * hf + 8 * q, 128));
        unpack8(u, x + 8 * q);
    }
}

// Multiply columns [64 hf, +64) of row r of a swizzled fp16 tile by w, in place.
__device__ __forceinline__ void scale_half_smem(uint8_t* tile, int r, int hf, float w) {
    float x[64];
    load_half_smem(tile, r, hf, x);
#pragma unroll
    for (int i = 0; i < 64; ++i) x[i] *= w;
    store_half_bf16<__half>(tile, r, hf, x);
}

__device__ __forceinline__ float dot64(const float (&x)[64], const float (&y)[64]) {
    float acc = 0.f;
#pragma unroll
    for (int i = 0; i < 64; ++i) acc = fmaf(x[i], y[i], acc);
    return acc;
}

// ---------------------------------------------------------------------------------------
// Chunk-start states of every chunk, walking each segment from its start state.
template <class SL>
__global__ void __launch_bounds__(256, 1) snap_fwd_tc(const __grid_constant__ CUtensorMap tk,
                                                       const __grid_constant__ CUtensorMap tv,
                                                       TcBwdArgs a) {
    const Shape s = a.s;
    const SL sl = slots_of<SL>(s);
    const int bh = blockIdx.x, seg = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nct = s.T / CT;
    const int c_begin = seg * TC_SEGC;
    const int nc = min(TC_SEGC, nct - c_begin);
    const int tid = threadIdx.x;
    const Role ro;
    const int row = ro.row, hf = ro.hf;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem);   // tma[2], mma[2]
    uint32_t* s_taddr = reinterpret_cast<uint32_t*>(smem + 64);
    uint8_t* tiles = smem + 1024;                         // [buf][A-> | K | V]
    if (tid == 0) {
        for (int i = 0; i < 4; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    if (ro.warp == 0) tmem_alloc(s_taddr, 256);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *s_taddr;
    const uint32_t tl = taddr + ((uint32_t)(32 * ro.q) << 16);
    auto issue_kv = [&](int c, int buf) {
        uint8_t* tK = tiles + (3 * buf + 1) * TILE;
        uint8_t* tV = tiles + (3 * buf + 2) * TILE;
        const int r0 = b * s.T + (c_begin + c) * CT;
        mbar_expect_tx(&bars[buf], 2 * TILE);
        tma_load_3d(tK, &tk, 0, h, r0, &bars[buf]);
        tma_load_3d(tK + TILE / 2, &tk, 64, h, r0, &bars[buf]);
        tma_load_3d(tV, &tv, 0, h, r0, &bars[buf]);
        tma_load_3d(tV + TILE / 2, &tv, 64, h, r0, &bars[buf]);
    };
    if (tid == 0) issue_kv(0, 0);
    {   // segment-start state into TMEM: thread half hf takes columns [128 hf, 128 hf + 128)
        const float* src = a.segS + (((size_t)bh * a.nseg + seg) * 128 + row) * 256 + 128 * hf;
#pragma unroll
        for (int q2 = 0; q2 < 2; ++q2) {
            float x[64];
#pragma unroll
            for (int i = 0; i < 64; i += 4) {
                const float4 f = *reinterpret_cast<const float4*>(src + 64 * q2 + i);
                x[i] = f.x; x[i + 1] = f.y; x[i + 2] = f.z; x[i + 3] = f.w;
            }
            tmem_st64(tl + 128 * hf + 64 * q2, x);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    bool ok = true;
    const uint32_t id_nn = idesc_f16(128, 128, 1, 1);
    for (int c = 0; c < nc; ++c) {
        const int buf = c & 1, cg = c_begin + c, t0 = cg * CT;
        if (c >= 1 && ok) ok = mbar_wait(&bars[2 + ((c - 1) & 1)], ((c - 1) >> 1) & 1);
        tc_fence_after();
        if (tid == 0 && ok && c + 1 < nc) issue_kv(c + 1, (c + 1) & 1);
        float lam, beta, g;
        load_gates_row(s, a, b, h, t0, row, lam, beta, g);
        const float gC = cum128(s, a.g, b, h, t0, t0 + CT - 1);
        {   // snapshot of this chunk's start state, then S <- gamma^C S
            __half* dst = a.snapF + (((size_t)bh * nct + cg) * 2 + hf) * 128 * 128 + row * 128;
            const float dC = ex2(gC * LOG2E);
#pragma unroll
            for (int q2 = 0; q2 < 2; ++q2) {
                float x[64];
                tmem_ld64(tl + 128 * hf + 64 * q2, x);
                store_global_half(dst + 64 * q2, x);
#pragma unroll
                for (int i = 0; i < 64; ++i) x[i] *= dC;
                tmem_st64(tl + 128 * hf + 64 * q2, x);
            }
        }
        write_vector_half<__half>(tiles + 3 * buf * TILE, row, hf, lam, beta * ex2((gC - g) * LOG2E),
                                  sl);
        if (ok) ok = mbar_wait(&bars[buf], (c >> 1) & 1);
        if (ok) {
            bf16_to_f16_half(tiles + (3 * buf + 1) * TILE, row, hf);
            bf16_to_f16_half(tiles + (3 * buf + 2) * TILE, row, hf);
        }
        fence_async_smem();
        tc_fence_before();
        ok = __syncthreads_and(ok);
        tc_fence_after();
        if (!ok) break;
        if (tid == 0) {
            {
                const uint32_t tA = smem_u32(tiles + 3 * buf * TILE);
                const uint32_t tK = smem_u32(tiles + (3 * buf + 1) * TILE);
                const uint32_t tV = smem_u32(tiles + (3 * buf + 2) * TILE);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    mma_bf16(taddr, mnmajor_desc(tA, 128, k), mnmajor_desc(tK, 128, k), id_nn, 1u);
                    mma_bf16(taddr + 128, mnmajor_desc(tA, 128, k), mnmajor_desc(tV, 128, k), id_nn, 1u);
                }
                mma_commit(&bars[2 + buf]);
            }
        }
    }
    if (ok) ok = mbar_wait(&bars[2 + ((nc - 1) & 1)], ((nc - 1) >> 1) & 1);
    ok = __syncthreads_and(ok);
    if (!ok && tid == 0) {
        flag_error(CYFA_ERR_TIMEOUT);
        for (int i = 0; i < 2; ++i) mbar_wait(&bars[i], 0);
    }
    tc_fence_before();
    __syncthreads();
    if (ro.warp == 0) tmem_dealloc(taddr, 256);
}

// ---------------------------------------------------------------------------------------
// Per chunk: recompute O', O''; dO''; middle-readout gradient; dO'; dq; per-token scalars.
// 512 threads: one row and one column quarter each (QRole).  Persistent: each CTA walks a
// contiguous range of (b*h, chunk) items; the next item's dO, Vbar (and M on a new head) are
// loaded into the tiles the current item has finished with after its dO' products, and its V
// after the last product, so an item starts with its operands mostly in place.  The six tiles
// change roles from item to item: (dO/Q, A, staging) <- (A, staging, dO/Q).
template <class SL>
__global__ void __launch_bounds__(512, 1) bwd_chunk1_tc(const __grid_constant__ CUtensorMap tq,
                                                         const __grid_constant__ CUtensorMap tk,
                                                         const __grid_constant__ CUtensorMap tv,
                                                         const __grid_constant__ CUtensorMap tdo,
                                                         const __grid_constant__ CUtensorMap tm,
                                                         const __grid_constant__ CUtensorMap tsf,
                                                         const __grid_constant__ CUtensorMap tmz,
                                                         const __grid_constant__ CUtensorMap tmp,
                                                         const __grid_constant__ CUtensorMap tmdy,
                                                         const __grid_constant__ CUtensorMap tmdl,
                                                         const __grid_constant__ CUtensorMap tdq,
                                                         TcBwdArgs a) {
    const Shape s = a.s;
    const SL sl = slots_of<SL>(s);
    const int nct = s.T / CT;
    const int NI = s.B * s.H * nct;   // items (b*h, chunk), b*h-major
    const int i0 = (int)((long long)NI * blockIdx.x / gridDim.x);
    const int i1 = (int)((long long)NI * (blockIdx.x + 1) / gridDim.x);
    const int tid = threadIdx.x;
    const QRole ro;
    const int row = ro.row, hf = ro.hf, u = ro.u, c0 = ro.c0, cq = ro.cq;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    // first operands (dO, Vbar, M), second operands (Q, K, Kbar), products, V
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem);
    uint32_t* s_taddr = reinterpret_cast<uint32_t*>(smem + 32);
    float* s_g2 = reinterpret_cast<float*>(smem + 64);              // [128]
    float* s_b = s_g2 + 128;                                        // [128] in-block decay factors
    float* s_red = s_b + 128;                                       // [2][4][128]
    float* s_gate = s_red + 1024;                                   // [5][128] next item's gates
    uint8_t* P = smem + 8192;                                       // six tiles
    int rL1 = 0, rA = 3, rS = 4;                                    // rotating roles
    uint8_t* T_K = P + 1 * TILE;      // V (first), then K
    uint8_t* T_KB = P + 2 * TILE;     // Vbar snapshot (first), then Kbar snapshot
    uint8_t* T_M = P + 5 * TILE;      // M = R Phi
    if (tid == 0) {
        for (int i = 0; i < 4; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    if (ro.warp == 0) tmem_alloc(s_taddr, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *s_taddr;
    const uint32_t tl = taddr + ((uint32_t)(32 * ro.q) << 16) + c0;
    const uint32_t X1 = 0, X2 = 128, X3 = 256, X4 = 384;
    const float scale = s.scale;
    const uint32_t id_kk = idesc_f16(128, 128, 0, 0), id_kn = idesc_f16(128, 128, 0, 1);
    bool ok = i0 < i1;
    // loads in flight (thread 0), for a clean stop after a failed wait
    // bits 0-2: a load on barrier 0 / 1 / 3 in flight; bits 4-6: the parity it completes
    uint32_t pend = 0;
    uint32_t ph = 0;                   // parity of the per-item barriers (0, 1, 3) of this item
    uint32_t mma_ph = 0;
    float g2 = 0.f;                    // this thread's log2-domain decay in the current item
    auto issue_first = [&](int item, uint8_t* tdO, uint8_t* tVb, bool with_m) {
        const int ibh = item / nct, icg = item - ibh * nct, ib = ibh / s.H, ih = ibh - ib * s.H;
        const int rtok = ib * s.T + icg * CT, srow = (ibh * nct + icg) * 2 * 128;
        mbar_expect_tx(&bars[0], (with_m ? 3 : 2) * TILE);
        tma_load_3d(tdO, &tdo, 0, ih, rtok, &bars[0]);
        tma_load_3d(tdO + TILE / 2, &tdo, 64, ih, rtok, &bars[0]);
        tma_load_2d(tVb, &tsf, 0, srow + 128, &bars[0]);
        tma_load_2d(tVb + TILE / 2, &tsf, 64, srow + 128, &bars[0]);
        if (with_m) {
            tma_load_2d(T_M, &tm, 0, ih * 128, &bars[0]);
            tma_load_2d(T_M + TILE / 2, &tm, 64, ih * 128, &bars[0]);
        }
        pend = (pend & ~0x11u) | 0x1u | ((uint32_t)((item - i0) & 1) << 4);
    };
    auto issue_v = [&](int item, uint8_t* tV) {
        const int ibh = item / nct, icg = item - ibh * nct, ib = ibh / s.H, ih = ibh - ib * s.H;
        mbar_expect_tx(&bars[3], TILE);
        tma_load_3d(tV, &tv, 0, ih, ib * s.T + icg * CT, &bars[3]);
        tma_load_3d(tV + TILE / 2, &tv, 64, ih, ib * s.T + icg * CT, &bars[3]);
        pend = (pend & ~0x44u) | 0x4u | ((uint32_t)((item - i0) & 1) << 6);
    };
    if (tid == 0 && ok) {
        issue_first(i0, P + rL1 * TILE, T_KB, true);
        issue_v(i0, T_K);
    }
    auto publish = [&]() {
        fence_async_smem();
        tc_fence_before();
        ok = __syncthreads_and(ok);
        tc_fence_after();
    };
    auto wait_mma = [&]() {
        if (ok) ok = mbar_wait(&bars[2], mma_ph);
        mma_ph ^= 1;
        tc_fence_after();
    };
    auto issuer = [&]() { return tid == 0 && ok; };
    // the staging tile (rows = the item's tokens) out to a [B*H*T][128] fp16 array by a TMA store
    // that runs beside the product reading the same tile; after the product, a barrier behind
    // thread 0's wait for the store's read guards the tile's next writes
    auto store_staged = [&](const CUtensorMap* map, const uint8_t* tile, int rowbh) {
        tma_store_2d(map, tile, 0, rowbh);
        tma_store_2d(map, tile + TILE / 2, 64, rowbh);
        bulk_commit();
    };
    auto staged_read = [&]() {   // every thread, after the product: the store has read the tile
        if (tid == 0) bulk_wait_read_all();
        __syncthreads();
    };
    // gates of the current item, and the next item's prefetched
    auto gate_index = [&](int item) {
        const int ibh = item / nct, icg = item - ibh * nct, ib = ibh / s.H, ih = ibh - ib * s.H;
        return ((size_t)ib * s.T + icg * CT + row) * s.H + ih;
    };
    // the gates of an item (clock, write strength, the two terms of the chunk-local decay) go to
    // s_gate by asynchronous copies, issued an epilogue ahead of their use (no registers held)
    auto stage_gates = [&](int item) {
        if (cq != 0) return;
        const int ibh = item / nct, icg = item - ibh * nct, ib = ibh / s.H, ih = ibh - ib * s.H;
        const size_t gi_ = ((size_t)ib * s.T + icg * CT + row) * s.H + ih;
        const float* src[5] = {a.lam + gi_, a.beta + gi_, a.g + gi_,
                               (s.Cg == 64 && row >= 64) ? a.g + ((size_t)ib * s.T + icg * CT + 63) * s.H + ih
                                                         : nullptr,
                               a.g + ((size_t)ib * s.T + icg * CT + (row | 15)) * s.H + ih};
#pragma unroll
        for (int k = 0; k < 5; ++k) {
            const uint32_t d = smem_u32(s_gate + 128 * k + row);
            if (src[k])
                asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(d), "l"(src[k]) : "memory");
            else
                s_gate[128 * k + row] = 0.f;
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    auto gates_landed = [&]() { asm volatile("cp.async.wait_group 0;" ::: "memory"); };
    if (ok) stage_gates(i0);
    gates_landed();
    __syncthreads();
    // x o Gamma (times mul) with the causal mask; columns are tokens of this chunk
    auto mask_scores = [&](float (&x)[32], float mul) {
        mask_decay_q(x, mul, row, ro.q, c0, g2, s_g2, s_b);
    };
    // sum / max of a per-thread partial over the four column quarters of this row (the same
    // order on every quarter, so all four get bit-identical results)
    int red_buf = 0;
    auto row_reduce = [&](float v, bool is_max) {
        float* r = s_red + 512 * red_buf;
        red_buf ^= 1;
        r[128 * cq + row] = v;
        __syncthreads();
        return is_max ? fmaxf(fmaxf(r[row], r[128 + row]), fmaxf(r[256 + row], r[384 + row]))
                      : (r[row] + r[128 + row]) + (r[256 + row] + r[384 + row]);
    };
    for (int it = i0; it < i1 && ok; ++it) {
        const int bh = it / nct, cg = it - bh * nct, b = bh / s.H, h = bh % s.H;
        const int t0 = cg * CT;
        const size_t gi = gate_index(it);
        const float lam = s_gate[row], beta = s_gate[128 + row];
        g2 = (s_gate[256 + row] + s_gate[384 + row]) * LOG2E;
        const float g2e = (s_gate[512 + row] + s_gate[384 + row]) * LOG2E;   // token row | 15
        uint8_t* T_L1 = P + rL1 * TILE;   // dO, then Q
        uint8_t* T_A = P + rA * TILE;     // write vectors (rows = tokens)
        uint8_t* T_S = P + rS * TILE;     // staging
        const int rowtok = b * s.T + t0, rowbh = bh * s.T + t0;
        const int snap_row = (bh * nct + cg) * 2 * 128;
        if (cq == 0) {
            s_g2[row] = g2;
            s_b[row] = ex2(g2e - g2);
        }
        if (ok) ok = mbar_wait(&bars[0], ph);
        if (tid == 0 && ok) pend &= ~0x1u;
        if (ok) ok = mbar_wait(&bars[3], ph);
        if (tid == 0 && ok) pend &= ~0x4u;
        if (ok) {   // dO and V: bf16 -> fp16
            bf16_to_f16_q(T_L1, row, c0);
            bf16_to_f16_q(T_K, row, c0);
        }
        // the previous item's dq store has read its staging tile, this item's T_A (written
        // after this barrier)
        if (tid == 0) bulk_wait_read_all();
        publish();
        if (!ok) break;
        const uint32_t uK = smem_u32(T_K), uKB = smem_u32(T_KB), uA = smem_u32(T_A), uM = smem_u32(T_M),
                       uS = smem_u32(T_S), uL1 = smem_u32(T_L1);
        const float gam = ex2(g2);
        float s1 = 0.f, s2 = 0.f, s3 = 0.f, s4 = 0.f;
        if (issuer()) {   // G1: X1 = dO V^T, X2 = dO Vbar^T
    #pragma unroll
            for (int k = 0; k < 8; ++k) {
                mma_bf16(taddr + X1, kmajor_desc(uL1, 128, k), kmajor_desc(uK, 128, k), id_kk, k > 0);
                mma_bf16(taddr + X2, kmajor_desc(uL1, 128, k), kmajor_desc(uKB, 128, k), id_kk, k > 0);
            }
            mma_commit(&bars[2]);
        }
        write_vector_q<__half>(T_A, row, hf, u, lam, beta, sl);   // while G1 runs
        wait_mma();
        if (issuer()) {   // dO, V and Vbar are consumed: Q, K and Kbar
            mbar_expect_tx(&bars[1], 3 * TILE);
            tma_load_3d(T_L1, &tq, 0, h, rowtok, &bars[1]);
            tma_load_3d(T_L1 + TILE / 2, &tq, 64, h, rowtok, &bars[1]);
            tma_load_3d(T_K, &tk, 0, h, rowtok, &bars[1]);
            tma_load_3d(T_K + TILE / 2, &tk, 64, h, rowtok, &bars[1]);
            tma_load_2d(T_KB, &tsf, 0, snap_row, &bars[1]);
            tma_load_2d(T_KB + TILE / 2, &tsf, 64, snap_row, &bars[1]);
            pend = (pend & ~0x22u) | 0x2u | (ph << 5);
        }
        {   // P4 = (dO V^T) o Gamma
            float x[32];
            tmem_ld16x2(tl + X1, x);
            mask_scores(x, 1.f);
            store_q<__half>(T_S, row, c0, x);
        }
        publish();
        if (issuer()) {   // G2: X3 = P4 A
    #pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X3, kmajor_desc(uS, 128, k), mnmajor_desc(uA, 128, k), id_kn, k > 0);
            mma_commit(&bars[2]);
        }
        wait_mma();
        {   // do'' = gamma (dO Vbar^T) + P4 A, kept in X2
            float x[32], y[32];
            tmem_ld16x2_pair(tl + X2, x, tl + X3, y);
            fma2_scalar(x, gam, y);
            tmem_st16x2(tl + X2, x);
            if (ok) ok = mbar_wait(&bars[1], ph);
            if (tid == 0 && ok) pend &= ~0x2u;
            if (ok) {   // Q and K: bf16 -> fp16
                bf16_to_f16_q(T_L1, row, c0);
                bf16_to_f16_q(T_K, row, c0);
            }
        }
        publish();
        if (issuer()) {   // G3: X1 = Q K^T, X3 = Q Kbar^T
    #pragma unroll
            for (int k = 0; k < 8; ++k) {
                mma_bf16(taddr + X1, kmajor_desc(uL1, 128, k), kmajor_desc(uK, 128, k), id_kk, k > 0);
                mma_bf16(taddr + X3, kmajor_desc(uL1, 128, k), kmajor_desc(uKB, 128, k), id_kk, k > 0);
            }
            mma_commit(&bars[2]);
        }
        wait_mma();
        {   // P1 = s (Q K^T) o Gamma
            float x[32];
            tmem_ld16x2(tl + X1, x);
            mask_scores(x, scale);
            store_q<__half>(T_S, row, c0, x);
        }
        publish();
        if (issuer()) {   // G4: X4 = P1 A
    #pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X4, kmajor_desc(uS, 128, k), mnmajor_desc(uA, 128, k), id_kn, k > 0);
            mma_commit(&bars[2]);
        }
        wait_mma();
        {   // z = U(lam) o', kept in X3
            float x[32], y[32];
            tmem_ld16x2_pair(tl + X3, x, tl + X4, y);
            const float f = scale * gam;
            fma2_scalar(x, f, y);
            rotate_q<1>(x, hf, u, lam, sl);
            store_q<__half>(T_S, row, c0, x);
            tmem_st16x2(tl + X3, x);
        }
        publish();
        if (issuer()) {   // G5: X1 = z M^T
            if (a.mZ) store_staged(&tmz, T_S, rowbh);
    #pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X1, kmajor_desc(uS, 128, k), kmajor_desc(uM, 128, k), id_kk, k > 0);
            mma_commit(&bars[2]);
        }
        wait_mma();
        if (a.mZ) staged_read();   // the staging tile is rewritten below (uniform branch)
        {   // p = softmax(l) over the m valid entries (the padding column is out), kept in X1
            float x[32];
            tmem_ld16x2(tl + X1, x);
            float mx = -INFINITY;
    #pragma unroll
            for (int i = 0; i < 32; ++i)
                if (!slot_off(c0, i, sl)) mx = fmaxf(mx, x[i]);
            mx = row_reduce(mx, true);
            float sum = 0.f;
    #pragma unroll
            for (int i = 0; i < 32; ++i) {
                x[i] = slot_off(c0, i, sl) ? 0.f : ex2((x[i] - mx) * LOG2E);
                sum += x[i];
            }
            const float inv = 1.f / row_reduce(sum, false);
    #pragma unroll
            for (int i = 0; i < 32; ++i) x[i] *= inv;
            store_q<__half>(T_S, row, c0, x);
            tmem_st16x2(tl + X1, x);
        }
        publish();
        if (issuer()) {   // G6: X4 = p M
            if (a.mP) store_staged(&tmp, T_S, rowbh);
    #pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X4, kmajor_desc(uS, 128, k), mnmajor_desc(uM, 128, k), id_kn, k > 0);
            mma_commit(&bars[2]);
        }
        wait_mma();
        if (a.mZ) staged_read();   // the staging tile is rewritten below (uniform branch)
        {   // o'' = U(-lam) (p M); scalars with do'' (o'' as stored in fp16); dy = U(lam) do''.
            // Eight rotation pairs at a time: cosine entries, then sine entries.
            QuarterAngles ang(lam, hf, u, sl);
            const float om1 = sl.omega1;
            const float wb = om1 * (float)(32 * hf + 16 * u + 1);   // pair frequency, first pair
            const bool dcq = (hf == 1 && u == 1);   // pair 15 of this quarter is the DC / padding
            __half* o2row = a.O2 + ((size_t)bh * s.T + t0 + row) * 128;
            uint32_t pc[8], ps[8];   // o'' packed: columns c0 .. c0 + 15 and c0 + 32 .. c0 + 47
    #pragma unroll
            for (int p8 = 0; p8 < 2; ++p8) {
                float o[16], gv[16];
                tmem_ld8x2_pair(tl + X4 + 8 * p8, o, tl + X2 + 8 * p8, gv);
    #pragma unroll
                for (int i = 0; i < 8; ++i) {
                    if (p8 + i > 0) ang.step();
                    const float c = ang.c, sn = ang.s;
                    const bool dc = dcq && p8 == 1 && i == 7;
                    const float xc = o[i], xs = o[8 + i];
                    o[i] = dc ? xc : c * xc + sn * xs;          // U(-lam)
                    o[8 + i] = dc ? 0.f : c * xs - sn * xc;
                    const float orc = round16<__half>(o[i]), ors = round16<__half>(o[8 + i]);
                    const float gc = gv[i], gs = gv[8 + i];
                    s1 = fmaf(orc, gc, fmaf(ors, gs, s1));
                    if (!dc)   // <o'', Omega do''>
                        s2 += (wb + om1 * (float)(8 * p8 + i)) * (ors * gc - orc * gs);
                    gv[i] = dc ? gc : c * gc - sn * gs;          // U(lam)
                    gv[8 + i] = dc ? 0.f : sn * gc + c * gs;
                }
    #pragma unroll
                for (int k = 0; k < 4; ++k) {
                    pc[4 * p8 + k] = pack_f16(o[2 * k], o[2 * k + 1]);
                    ps[4 * p8 + k] = pack_f16(o[8 + 2 * k], o[9 + 2 * k]);
                }
                store8x2<__half>(T_S, row, c0 + 8 * p8, gv);
            }
            st_global_v8(o2row + c0, pc);
            st_global_v8(o2row + c0 + 32, ps);
        }
        publish();
        if (issuer()) {   // G7: X4 = dy M^T = M dy
            if (a.mDY) store_staged(&tmdy, T_S, rowbh);
    #pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X4, kmajor_desc(uS, 128, k), kmajor_desc(uM, 128, k), id_kk, k > 0);
            mma_commit(&bars[2]);
        }
        wait_mma();
        if (a.mZ) staged_read();   // the staging tile is rewritten below (uniform branch)
        {   // dl = p o (dp - <p, dp>)
            float p[32], dp[32];
            tmem_ld16x2_pair(tl + X1, p, tl + X4, dp);
            const float pdp = row_reduce(dot32(p, dp), false);
    #pragma unroll
            for (int i = 0; i < 32; ++i) p[i] = p[i] * (dp[i] - pdp);
            store_q<__half>(T_S, row, c0, p);
        }
        publish();
        if (issuer()) {   // G8: X2 = dl M = M^T dl
            if (a.mDL) store_staged(&tmdl, T_S, rowbh);
    #pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X2, kmajor_desc(uS, 128, k), mnmajor_desc(uM, 128, k), id_kn, k > 0);
            mma_commit(&bars[2]);
        }
        wait_mma();
        if (a.mZ) staged_read();   // the staging tile is rewritten below (uniform branch)
        {   // do' = U(-lam) dz; <do', Omega o'> with do' as stored in fp16 (= <dz, Omega z> exactly)
            QuarterAngles ang(lam, hf, u, sl);
            const float om1 = sl.omega1;
            const float wb = om1 * (float)(32 * hf + 16 * u + 1);   // pair frequency, first pair
            const bool dcq = (hf == 1 && u == 1);
            __half* d1row = a.DO1 + ((size_t)bh * s.T + t0 + row) * 128;
            uint32_t pc[8], ps[8];   // do' packed: columns c0 .. c0 + 15 and c0 + 32 .. c0 + 47
    #pragma unroll
            for (int p8 = 0; p8 < 2; ++p8) {
                float dz[16], z[16];
                tmem_ld8x2_pair(tl + X2 + 8 * p8, dz, tl + X3 + 8 * p8, z);
    #pragma unroll
                for (int i = 0; i < 8; ++i) {
                    if (p8 + i > 0) ang.step();
                    const float c = ang.c, sn = ang.s;
                    const bool dc = dcq && p8 == 1 && i == 7;
                    const float xc = dz[i], xs = dz[8 + i];
                    dz[i] = dc ? xc : c * xc + sn * xs;         // U(-lam)
                    dz[8 + i] = dc ? 0.f : c * xs - sn * xc;
                    if (!dc) {   // o' = U(-lam) z
                        const float zc = c * z[i] + sn * z[8 + i], zs = c * z[8 + i] - sn * z[i];
                        s3 += (wb + om1 * (float)(8 * p8 + i)) *
                              (round16<__half>(dz[8 + i]) * zc - round16<__half>(dz[i]) * zs);
                    }
                }
                store8x2<__half>(T_S, row, c0 + 8 * p8, dz);
    #pragma unroll
                for (int k = 0; k < 4; ++k) {
                    pc[4 * p8 + k] = pack_f16(dz[2 * k], dz[2 * k + 1]);
                    ps[4 * p8 + k] = pack_f16(dz[8 + 2 * k], dz[9 + 2 * k]);
                }
            }
            st_global_v8(d1row + c0, pc);
            st_global_v8(d1row + c0 + 32, ps);
        }
        publish();
        if (issuer()) {   // G9: X1 = dO' A^T, X3 = dO' Kbar
    #pragma unroll
            for (int k = 0; k < 8; ++k) {
                mma_bf16(taddr + X1, kmajor_desc(uS, 128, k), kmajor_desc(uA, 128, k), id_kk, k > 0);
                mma_bf16(taddr + X3, kmajor_desc(uS, 128, k), mnmajor_desc(uKB, 128, k), id_kn, k > 0);
            }
            mma_commit(&bars[2]);
        }
        wait_mma();
        if (issuer() && it + 1 < i1) {
            issue_first(it + 1, T_A, T_KB, (it + 1) / nct % s.H != h);
            // the next item's V into L2: its load waits for this item's last product
            const int nbh = (it + 1) / nct, ncg = (it + 1) - nbh * nct, nb = nbh / s.H;
            tma_prefetch_3d(&tv, 0, nbh - nb * s.H, nb * s.T + ncg * CT);
            tma_prefetch_3d(&tv, 64, nbh - nb * s.H, nb * s.T + ncg * CT);
        }
        if (it + 1 < i1) stage_gates(it + 1);   // the next item's gates, an epilogue ahead
        {   // P3 = s (dO' A^T) o Gamma
            float x[32];
            tmem_ld16x2(tl + X1, x);
            mask_scores(x, scale);
            store_q<__half>(T_S, row, c0, x);
        }
        publish();
        if (issuer()) {   // G10: X4 = P3 K
    #pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X4, kmajor_desc(uS, 128, k), mnmajor_desc(uK, 128, k), id_kn, k > 0);
            mma_commit(&bars[2]);
        }
        wait_mma();
        if (issuer() && it + 1 < i1) issue_v(it + 1, T_K);
        if (ok) {   // dq = s gamma (dO' Kbar) + P3 K  (P3 carries s) ; <q, dq> = <q~, dq~>
            float x[32], y[32];
            tmem_ld16x2_pair(tl + X3, x, tl + X4, y);
            const float f = scale * gam;
            fma2_scalar(x, f, y);
            load_q(T_L1, row, c0, y);
            s4 = dot32(y, x);
            // dq leaves through the staging tile (P3 is consumed) by a TMA store
            store_q<__nv_bfloat16>(T_S, row, c0, x);
            fence_async_smem();
        }
        gates_landed();   // the next item's gates, visible after the barriers below
        {
            const float dG = row_reduce(s1 + s4, false);
            if (issuer()) {   // the staged dq rows are complete after the reduction's barrier
                tma_store_3d(&tdq, T_S, 0, h, rowtok);
                tma_store_3d(&tdq, T_S + TILE / 2, 64, h, rowtok);
                bulk_commit();
            }
            const float dL = row_reduce(s3 + s2, false);
            if (cq == 0 && ok) {
                const size_t BTH = (size_t)s.B * s.T * s.H;
                a.tok[gi] = dG;
                a.tok[BTH + gi] = dL;
            }
        }
        ph ^= 1;
        {   // roles of the next item
            const int l1 = rL1;
            rL1 = rA;
            rA = rS;
            rS = l1;
        }
    }
    ok = __syncthreads_and(ok);
    if (!ok && tid == 0) {
        flag_error(CYFA_ERR_TIMEOUT);
        // let copies still in flight land before the shared memory is released
        if (pend & 0x1u) mbar_wait(&bars[0], (pend >> 4) & 1);
        if (pend & 0x2u) mbar_wait(&bars[1], (pend >> 5) & 1);
        if (pend & 0x4u) mbar_wait(&bars[3], (pend >> 6) & 1);
    }
    if (tid == 0) bulk_wait_all();
    tc_fence_before();
    __syncthreads();
    if (ro.warp == 0) tmem_dealloc(taddr, 512);
}

// ---------------------------------------------------------------------------------------
// Adjoint states of the reversed recurrence, per segment.  SNAP = false: the segment's own
// contribution  dD = sum_r exp(G_r - G_start) [dO'_r q~_r^T | o''_r dO_r^T]  (into segD);
// SNAP = true: walk the segment backwards from its end adjoint (segD after the reverse scan),
// storing before each chunk the adjoint of that chunk's end state, then
// D <- gamma^C D + sum_r gamma^r [...].  The K part (dO', q~) and the V part (o'', dO) run one
// after the other with double-buffered tiles.  In the SNAP walk the chunk-start state S of
// the forward (for the boundary terms of the gate gradients) arrives by TMA with the operand
// tiles, and the adjoint snapshot leaves through the same shared tile by a TMA store.
template <bool SNAP, class SL>
__global__ void __launch_bounds__(256, 1) adj_walk_tc(const __grid_constant__ CUtensorMap tdo1,
                                                       const __grid_constant__ CUtensorMap to2,
                                                       const __grid_constant__ CUtensorMap tq,
                                                       const __grid_constant__ CUtensorMap tdo,
                                                       const __grid_constant__ CUtensorMap tsf,
                                                       const __grid_constant__ CUtensorMap tsa,
                                                       TcBwdArgs a) {
    const Shape s = a.s;
    const SL sl = slots_of<SL>(s);
    const int bh = blockIdx.x, seg = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nct = s.T / CT;
    const int c_begin = seg * TC_SEGC;
    const int nc = min(TC_SEGC, nct - c_begin);
    const int tid = threadIdx.x;
    const Role ro;
    const int row = ro.row, hf = ro.hf;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem);   // tma[2], mma[2]
    uint32_t* s_taddr = reinterpret_cast<uint32_t*>(smem + 64);
    float* s_tot = reinterpret_cast<float*>(smem + 128);   // [TC_SEGC]
    float* s_pre = s_tot + TC_SEGC;                         // [TC_SEGC]
    float* s_bnd = s_pre + TC_SEGC;                         // [TC_SEGC][2]
    float* s_gs = reinterpret_cast<float*>(smem + 1024);    // [TC_SEGC * CT] chunk-local decays
    constexpr int NT = SNAP ? 3 : 2;                       // tiles per buffer
    constexpr int NB = SNAP ? 2 : 3;                       // buffers: loads run NB - 1 chunks ahead
    uint8_t* tiles = smem + 1024 + 4 * TC_SEGC * CT;       // [buf][X | Y (| S)]
    const int total = 2 * nc;   // iterations: part 0 (K) chunks, then part 1 (V) chunks
    auto chunk_of = [&](int it) {
        const int i = it % nc;
        return SNAP ? nc - 1 - i : i;
    };
    int issued = 0, landed = 0;   // thread 0: loads issued / seen complete
    auto issue = [&](int it) {
        const int part = it / nc, c = chunk_of(it), buf = it % NB;
        ++issued;
        uint8_t* tX = tiles + (NT * buf) * TILE;
        uint8_t* tY = tX + TILE;
        const int t0 = (c_begin + c) * CT;
        const int xrow = bh * s.T + t0, yrow = b * s.T + t0;
        const CUtensorMap* mx = part == 0 ? &tdo1 : &to2;
        const CUtensorMap* my = part == 0 ? &tq : &tdo;
        mbar_expect_tx(&bars[buf], NT * TILE);
        tma_load_2d(tX, mx, 0, xrow, &bars[buf]);
        tma_load_2d(tX + TILE / 2, mx, 64, xrow, &bars[buf]);
        tma_load_3d(tY, my, 0, h, yrow, &bars[buf]);
        tma_load_3d(tY + TILE / 2, my, 64, h, yrow, &bars[buf]);
        if (SNAP) {
            uint8_t* tS = tX + 2 * TILE;
            const int srow = ((bh * nct + c_begin + c) * 2 + part) * 128;
            tma_load_2d(tS, &tsf, 0, srow, &bars[buf]);
            tma_load_2d(tS + TILE / 2, &tsf, 64, srow, &bars[buf]);
        }
    };
    auto prefetch = [&](int it) {   // the tiles of iteration it into L2
        const int part = it / nc, c = chunk_of(it);
        const int t0 = (c_begin + c) * CT;
        const int xrow = bh * s.T + t0, yrow = b * s.T + t0;
        const CUtensorMap* mx = part == 0 ? &tdo1 : &to2;
        const CUtensorMap* my = part == 0 ? &tq : &tdo;
#pragma unroll
        for (int x = 0; x < 128; x += 64) {
            tma_prefetch_2d(mx, x, xrow);
            tma_prefetch_3d(my, x, h, yrow);
            if (SNAP) tma_prefetch_2d(&tsf, x, ((bh * nct + c_begin + c) * 2 + part) * 128);
        }
    };
    if (tid == 0) {   // the first operand tiles are on their way while the decays load
        for (int i = 0; i < 2 * NB; ++i) mbar_init(&bars[i], 1);   // tma[NB], mma[NB]
        fence_mbar_init();
        for (int i = 0; i < NB - 1 && i < total; ++i) issue(i);
        if (NB - 1 < total) prefetch(NB - 1);
    }
    {   // every token's decay, loaded once: all of a thread's loads in flight together
        constexpr int NPT = TC_SEGC * CT / 256;
        float v[NPT], w[NPT];
#pragma unroll
        for (int k = 0; k < NPT; ++k) {
            const int i = tid + 256 * k;
            const int t0 = (c_begin + i / CT) * CT, t = t0 + i % CT;
            v[k] = i < nc * CT ? a.g[((size_t)b * s.T + t) * s.H + h] : 0.f;
            w[k] = (i < nc * CT && s.Cg == 64 && t - t0 >= 64) ? a.g[((size_t)b * s.T + t0 + 63) * s.H + h] : 0.f;
        }
#pragma unroll
        for (int k = 0; k < NPT; ++k)
            if (tid + 256 * k < nc * CT) s_gs[tid + 256 * k] = v[k] + w[k];   // cum128
    }
    if (ro.warp == 0) tmem_alloc(s_taddr, 256);
    if (tid < nc) {
        const int t0 = (c_begin + tid) * CT;
        s_tot[tid] = cum128(s, a.g, b, h, t0, t0 + CT - 1);
        s_bnd[2 * tid] = 0.f;
        s_bnd[2 * tid + 1] = 0.f;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *s_taddr;
    const uint32_t tl = taddr + ((uint32_t)(32 * ro.q) << 16);
    if (tid == 0) {
        float acc = 0.f;
        for (int c = 0; c < nc; ++c) {
            s_pre[c] = acc;
            acc += s_tot[c];
        }
    }
    if (SNAP) {   // end-of-segment adjoint into TMEM
        const float* src = a.segD + (((size_t)bh * a.nseg + seg) * 128 + row) * 256 + 128 * hf;
#pragma unroll
        for (int q2 = 0; q2 < 2; ++q2) {
            float x[64];
#pragma unroll
            for (int i = 0; i < 64; i += 4) {
                const float4 f = *reinterpret_cast<const float4*>(src + 64 * q2 + i);
                x[i] = f.x; x[i + 1] = f.y; x[i + 2] = f.z; x[i + 3] = f.w;
            }
            tmem_st64(tl + 128 * hf + 64 * q2, x);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    bool ok = true;
    const uint32_t id_nn = idesc_f16(128, 128, 1, 1);
    for (int it = 0; it < total; ++it) {
        const int part = it / nc, c = chunk_of(it), buf = it % NB;
        const int cg = c_begin + c;
        // product it - 1 must be complete before its buffer is refilled (and, in the SNAP walk,
        // before D is read); the refill goes out right after this chunk's operand rows are
        // prepared, which overlaps product it - 1
        auto refill = [&]() {
            if (it >= 1 && ok) ok = mbar_wait(&bars[NB + (it - 1) % NB], ((it - 1) / NB) & 1);
            tc_fence_after();
            if (tid == 0 && ok && it + NB - 1 < total) {
                if (SNAP) bulk_wait_read_all();   // the other buffer's S tile may be a store's source
                issue(it + NB - 1);
                if (it + NB < total) prefetch(it + NB);
            }
        };
        if (ok) ok = mbar_wait(&bars[buf], (it / NB) & 1);
        if (tid == 0 && ok) ++landed;
        const float g = s_gs[c * CT + row];
        uint8_t* tX = tiles + (NT * buf) * TILE;
        // this chunk's operand rows (its own buffer) are prepared while product it - 1 runs
        float w = SNAP ? ex2(g * LOG2E) : ex2((s_pre[c] + g) * LOG2E);
        if (part == 0) w *= s.scale;   // q~ = s q
        if (ok) {
            scale_half_smem(tX, row, hf, w);
            bf16_to_f16_half(tX + TILE, row, hf);   // q or dO
        }
        refill();
        if (SNAP) {
            // adjoint of this chunk's end state, then D <- gamma^C D (this part's 128 columns)
            uint8_t* tS = tX + 2 * TILE;
            const float dC = ex2(s_tot[c] * LOG2E);
            float x[64];
            tmem_ld64(tl + 128 * part + 64 * hf, x);
            {
                // gamma^C <D, S> and gamma^C <D, Omega S> with S this chunk's start state (the
                // chunk's own writes enter through the inter-chunk column terms of
                // bwd_chunk2_tc); this thread's row and 64 columns
                const int l = row & 63, jj = l & 31, j = 32 * (row >> 6) + jj + 1;
                const bool paired = j <= sl.npair;
                const int partner = (l >= 32) ? row - 32 : row + 32;
                const float f = paired ? ((l >= 32) ? 1.f : -1.f) * sl.omega1 * (float)j : 0.f;
                float sr[64], sp[64];
                load_half_smem(tS, row, hf, sr);
                load_half_smem(tS, paired ? partner : row, hf, sp);
                float bG = dC * dot64(x, sr), bL = dC * f * dot64(x, sp);
                bG = warp_sum(bG);
                bL = warp_sum(bL);
                if (ro.lane == 0) {
                    atomicAdd(&s_bnd[2 * c], bG);
                    atomicAdd(&s_bnd[2 * c + 1], bL);
                }
            }
            __syncthreads();   // the S tile is read: it now stages the snapshot for its TMA store
            store_half_bf16<__half>(tS, row, hf, x);
#pragma unroll
            for (int i = 0; i < 64; ++i) x[i] *= dC;
            tmem_st64(tl + 128 * part + 64 * hf, x);
        }

        fence_async_smem();
        tc_fence_before();
        ok = __syncthreads_and(ok);
        tc_fence_after();
        if (!ok) break;
        if (tid == 0) {
            if (SNAP) {
                const int arow = ((bh * nct + cg) * 2 + part) * 128;
                tma_store_2d(&tsa, tX + 2 * TILE, 0, arow);
                tma_store_2d(&tsa, tX + 2 * TILE + TILE / 2, 64, arow);
                bulk_commit();
            }
            const uint32_t uX = smem_u32(tX);
            const uint32_t uY = smem_u32(tX + TILE);
            const bool first = !SNAP && (it % nc) == 0;
#pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + 128 * part, mnmajor_desc(uX, 128, k), mnmajor_desc(uY, 128, k),
                         id_nn, (first && k == 0) ? 0u : 1u);
            mma_commit(&bars[NB + buf]);
        }
    }
    if (ok) ok = mbar_wait(&bars[NB + (total - 1) % NB], ((total - 1) / NB) & 1);
    tc_fence_after();
    ok = __syncthreads_and(ok);
    if (SNAP && ok && tid < nc) {
        float* dst = a.bnd + ((size_t)bh * nct + c_begin + tid) * 2;
        dst[0] = s_bnd[2 * tid];
        dst[1] = s_bnd[2 * tid + 1];
    }
    if (ok && !SNAP) {   // the segment's contribution out through the (now idle) tiles, coalesced
        float* stage = reinterpret_cast<float*>(tiles);
#pragma unroll
        for (int q2 = 0; q2 < 2; ++q2) {
            float x[64];
            tmem_ld64(tl + 128 * hf + 64 * q2, x);
#pragma unroll
            for (int i = 0; i < 64; i += 4)
                *reinterpret_cast<float4*>(stage + row * STAGE_LD + 128 * hf + 64 * q2 + i) =
                    make_float4(x[i], x[i + 1], x[i + 2], x[i + 3]);
        }
        __syncthreads();
        stage_to_global_128x256(a.segD + ((size_t)bh * a.nseg + seg) * 128 * 256, stage, tid, 256);
    }
    if (!ok && tid == 0) {
        flag_error(CYFA_ERR_TIMEOUT);
        // let every copy issued so far land before the shared memory is released
        for (int i = landed; i < issued; ++i) mbar_wait(&bars[i % NB], (i / NB) & 1);
    }
    if (SNAP && tid == 0) bulk_wait_all();
    tc_fence_before();
    __syncthreads();
    if (ro.warp == 0) tmem_dealloc(taddr, 256);
}

// End-of-segment adjoints: D_end(last) = 0, D_end(j-1) = exp(G_j) D_end(j) + dD(j), in place.
__global__ void __launch_bounds__(256) seg_scan_rev_kernel(TcBwdArgs a) {
    const int bh = blockIdx.y;
    const int e = blockIdx.x * 256 + threadIdx.x;
    float* base = a.segD + (size_t)bh * a.nseg * 128 * 256 + e;
    const float* G = a.segG + (size_t)bh * a.nseg;
    float cur = 0.f;
    for (int j1 = a.nseg - 1; j1 >= 0; j1 -= 32) {
        float d[32], gj[32];   // all loads first: the stores below may alias them
#pragma unroll
        for (int u = 0; u < 32; ++u) {
            const int j = j1 - u;
            d[u] = j >= 0 ? base[(size_t)j * 128 * 256] : 0.f;
            gj[u] = j >= 0 ? G[j] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 32; ++u) {
            const int j = j1 - u;
            if (j >= 0) {
                base[(size_t)j * 128 * 256] = cur;
                cur = expf(gj[u]) * cur + d[u];
            }
        }
    }
}

// ---------------------------------------------------------------------------------------
// Per chunk: dK, dV, dA (both passes) and the column-side gate scalars, from the adjoint
// snapshot.  The intra-chunk and the inter-chunk parts of dA are kept apart (X3 / X4) so that
// the gate kernel can pair every intra-chunk term with its row-side twin from bwd_chunk1_tc,
// which uses bit-identical score matrices and roundings.  512 threads (QRole).  Persistent over
// (b*h, chunk) items like bwd_chunk1_tc: the next item's V goes into the write-vector tile once
// dO' A^T has read it, its dO into the Q tile after Q K^T, its O'' and D^V after the last
// products; the write-vector tile and the V / K tile swap roles from item to item.
template <class SL>
__global__ void __launch_bounds__(512, 1) bwd_chunk2_tc(const __grid_constant__ CUtensorMap tq,
                                                         const __grid_constant__ CUtensorMap tk,
                                                         const __grid_constant__ CUtensorMap tv,
                                                         const __grid_constant__ CUtensorMap tdo,
                                                         const __grid_constant__ CUtensorMap to2,
                                                         const __grid_constant__ CUtensorMap tdo1,
                                                         const __grid_constant__ CUtensorMap tsa,
                                                         const __grid_constant__ CUtensorMap tdk,
                                                         const __grid_constant__ CUtensorMap tdv,
                                                         TcBwdArgs a) {
    const Shape s = a.s;
    const SL sl = slots_of<SL>(s);
    const int nct = s.T / CT;
    const int NI = s.B * s.H * nct;
    const int i0 = (int)((long long)NI * blockIdx.x / gridDim.x);
    const int i1 = (int)((long long)NI * (blockIdx.x + 1) / gridDim.x);
    const int tid = threadIdx.x;
    const QRole ro;
    const int row = ro.row, hf = ro.hf, u = ro.u, c0 = ro.c0, cq = ro.cq;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    // 0: O'' + D^V, 1: K, 2: dO', 3: Q + D^K, 4: products, 5: V, 6: dO
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem);
    uint32_t* s_taddr = reinterpret_cast<uint32_t*>(smem + 64);
    float* s_g2 = reinterpret_cast<float*>(smem + 128);
    float* s_b = s_g2 + 128;          // [128] in-block decay factors
    uint8_t* P = smem + 2048;
    int rA = 0, rL2 = 4;              // the write-vector tile and the V / K tile swap each item
    uint8_t* T_AS = P + 1 * TILE;     // write vectors scaled by gamma^C / gamma^s
    uint8_t* T_S = P + 2 * TILE;      // staging
    uint8_t* L1 = P + 3 * TILE;       // dO, then Q
    uint8_t* L3 = P + 5 * TILE;       // O'', then dO'
    uint8_t* L4 = P + 6 * TILE;       // D^V, then D^K
    if (tid == 0) {
        for (int i = 0; i < 7; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
    }
    if (ro.warp == 0) tmem_alloc(s_taddr, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *s_taddr;
    const uint32_t tl = taddr + ((uint32_t)(32 * ro.q) << 16) + c0;
    const uint32_t X1 = 0, X2 = 128, X3 = 256, X4 = 384;
    const float scale = s.scale;
    const uint32_t id_kk = idesc_f16(128, 128, 0, 0), id_kn = idesc_f16(128, 128, 0, 1),
                   id_nn = idesc_f16(128, 128, 1, 1);
    bool ok = i0 < i1;
    // thread 0: bit k set = a load on barrier k in flight (its parity in bit 8 + k)
    uint32_t pend = 0;
    uint32_t ph = 0, mma_ph = 0;
    float g2 = 0.f;
    auto item_rows = [&](int item, int& ih, int& rtok, int& rbh, int& srow) {
        const int ibh = item / nct, icg = item - ibh * nct, ib = ibh / s.H;
        ih = ibh - ib * s.H;
        rtok = ib * s.T + icg * CT;
        rbh = ibh * s.T + icg * CT;
        srow = (ibh * nct + icg) * 2 * 128;
    };
    auto mark = [&](int k, int item) {
        pend = (pend & ~((1u << k) | (1u << (8 + k)))) | (1u << k) | ((uint32_t)((item - i0) & 1) << (8 + k));
    };
    auto issue_first = [&](int item, uint8_t* tO2, uint8_t* tDV) {
        int ih, rtok, rbh, srow;
        item_rows(item, ih, rtok, rbh, srow);
        mbar_expect_tx(&bars[0], 2 * TILE);
        tma_load_2d(tO2, &to2, 0, rbh, &bars[0]);
        tma_load_2d(tO2 + TILE / 2, &to2, 64, rbh, &bars[0]);
        tma_load_2d(tDV, &tsa, 0, srow + 128, &bars[0]);
        tma_load_2d(tDV + TILE / 2, &tsa, 64, srow + 128, &bars[0]);
        mark(0, item);
    };
    auto issue_v = [&](int item, uint8_t* tV) {
        int ih, rtok, rbh, srow;
        item_rows(item, ih, rtok, rbh, srow);
        mbar_expect_tx(&bars[5], TILE);
        tma_load_3d(tV, &tv, 0, ih, rtok, &bars[5]);
        tma_load_3d(tV + TILE / 2, &tv, 64, ih, rtok, &bars[5]);
        mark(5, item);
    };
    auto issue_do = [&](int item, uint8_t* tD) {
        int ih, rtok, rbh, srow;
        item_rows(item, ih, rtok, rbh, srow);
        mbar_expect_tx(&bars[6], TILE);
        tma_load_3d(tD, &tdo, 0, ih, rtok, &bars[6]);
        tma_load_3d(tD + TILE / 2, &tdo, 64, ih, rtok, &bars[6]);
        mark(6, item);
    };
    if (tid == 0 && ok) {
        issue_first(i0, L3, L4);
        issue_v(i0, P + rL2 * TILE);
        issue_do(i0, L1);
    }
    auto publish = [&]() {
        fence_async_smem();
        tc_fence_before();
        ok = __syncthreads_and(ok);
        tc_fence_after();
    };
    auto wait_mma = [&]() {
        if (ok) ok = mbar_wait(&bars[4], mma_ph);
        mma_ph ^= 1;
        tc_fence_after();
    };
    auto issuer = [&]() { return tid == 0 && ok; };
    auto mask_scores = [&](float (&x)[32], float mul) {
        mask_decay_q(x, mul, row, ro.q, c0, g2, s_g2, s_b);
    };
    for (int it = i0; it < i1 && ok; ++it) {
        const int bh = it / nct, cg = it - bh * nct, b = bh / s.H, h = bh % s.H;
        const int t0 = cg * CT;
        const size_t gi = ((size_t)b * s.T + t0 + row) * s.H + h;
        // gates: loaded while this item's first tiles land
        const float lam = a.lam[gi], beta = a.beta[gi];
        g2 = cum128(s, a.g, b, h, t0, t0 + row) * LOG2E;
        const float g2e = cum128(s, a.g, b, h, t0, t0 + (row | 15)) * LOG2E;
        const float g2C = cum128(s, a.g, b, h, t0, t0 + CT - 1) * LOG2E;
        const float fw = ex2(g2C - g2);
        uint8_t* T_A = P + rA * TILE;     // write vectors a (fp16)
        uint8_t* L2 = P + rL2 * TILE;     // V (-> V->), then K (-> K->)
        const int rowtok = b * s.T + t0, rowbh = bh * s.T + t0;
        const int snap_row = (bh * nct + cg) * 2 * 128;
        if (cq == 0) {
            s_g2[row] = g2;
            s_b[row] = ex2(g2e - g2);
        }
        if (ok) ok = mbar_wait(&bars[0], ph) && mbar_wait(&bars[5], ph) && mbar_wait(&bars[6], ph);
        if (tid == 0 && ok) pend &= ~0x61u;
        if (ok) {   // dO and V: bf16 -> fp16
            bf16_to_f16_q(L1, row, c0);
            bf16_to_f16_q(L2, row, c0);
        }
        publish();
        if (!ok) break;
        const uint32_t uA = smem_u32(T_A), uAS = smem_u32(T_AS), uS = smem_u32(T_S),
                       u1 = smem_u32(L1), u2 = smem_u32(L2), u3 = smem_u32(L3), u4 = smem_u32(L4);
        float cG = 0.f;
        if (issuer()) {   // X1 = dO V^T
    #pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X1, kmajor_desc(u1, 128, k), kmajor_desc(u2, 128, k), id_kk, k > 0);
            // the P4 epilogue rewrites T_S once this completes: the previous item's dk store must
            // have read it first (the commit is only issued after that)
            bulk_wait_read_all();
            mma_commit(&bars[4]);
        }
        {   // while it runs: the write vectors and their copies scaled by gamma^C / gamma^s
            float x[32];
            write_vector_q_vals(x, hf, u, lam, beta, sl);
            store_q<__half>(T_A, row, c0, x);
#pragma unroll
            for (int i = 0; i < 32; ++i) x[i] *= fw;
            store_q<__half>(T_AS, row, c0, x);
        }
        wait_mma();
        {   // P4 = (dO V^T) o Gamma ; V -> V-> (rows scaled by gamma^C / gamma^s)
            float x[32];
            tmem_ld16x2(tl + X1, x);
            mask_scores(x, 1.f);
            store_q<__half>(T_S, row, c0, x);
            if (ok) scale_q(L2, row, c0, fw);
        }
        publish();
        if (issuer()) {   // X3 = P4^T O'' ; X4 = V-> D^V^T ; X1 = O'' A^T
    #pragma unroll
            for (int k = 0; k < 8; ++k) {
                mma_bf16(taddr + X3, mnmajor_desc(uS, 128, k), mnmajor_desc(u3, 128, k), id_nn, k > 0);
                mma_bf16(taddr + X4, kmajor_desc(u2, 128, k), kmajor_desc(u4, 128, k), id_kk, k > 0);
                mma_bf16(taddr + X1, kmajor_desc(u3, 128, k), kmajor_desc(uA, 128, k), id_kk, k > 0);
            }
            mma_commit(&bars[4]);
        }
        wait_mma();
        if (issuer()) {   // V and O'' are consumed: K, dO'
            mbar_expect_tx(&bars[1], TILE);
            tma_load_3d(L2, &tk, 0, h, rowtok, &bars[1]);
            tma_load_3d(L2 + TILE / 2, &tk, 64, h, rowtok, &bars[1]);
            mbar_expect_tx(&bars[2], TILE);
            tma_load_2d(L3, &tdo1, 0, rowbh, &bars[2]);
            tma_load_2d(L3 + TILE / 2, &tdo1, 64, rowbh, &bars[2]);
            mark(1, it);
            mark(2, it);
        }
        {   // <a, (P4^T O'')_t> ; P2 = (O'' A^T) o Gamma
            float x[32], av[32];
            tmem_ld16x2(tl + X3, x);
            load_q(T_A, row, c0, av);   // the fp16 write vector entries, as the MMAs see them
            cG = dot32(av, x);
            tmem_ld16x2(tl + X1, x);
            mask_scores(x, 1.f);
            store_q<__half>(T_S, row, c0, x);
        }
        publish();
        if (issuer()) {   // X2 = P2^T dO + A-> D^V  (dv)
    #pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X2, mnmajor_desc(uS, 128, k), mnmajor_desc(u1, 128, k), id_nn, k > 0);
    #pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr + X2, kmajor_desc(uAS, 128, k), mnmajor_desc(u4, 128, k), id_kn, 1u);
            mma_commit(&bars[4]);
        }
        wait_mma();
        if (issuer()) {   // dO and D^V are consumed: Q, D^K
            mbar_expect_tx(&bars[3], 2 * TILE);
            tma_load_3d(L1, &tq, 0, h, rowtok, &bars[3]);
            tma_load_3d(L1 + TILE / 2, &tq, 64, h, rowtok, &bars[3]);
            tma_load_2d(L4, &tsa, 0, snap_row, &bars[3]);
            tma_load_2d(L4 + TILE / 2, &tsa, 64, snap_row, &bars[3]);
            mark(3, it);
        }
        if (ok) {   // dv, staged in T_S (P2 is consumed) for a TMA store
            float x[32];
            tmem_ld16x2(tl + X2, x);
            store_q<__nv_bfloat16>(T_S, row, c0, x);
        }
        publish();
        if (issuer()) {
            tma_store_3d(&tdv, T_S, 0, h, rowtok);
            tma_store_3d(&tdv, T_S + TILE / 2, 64, h, rowtok);
            bulk_commit();
        }
        if (issuer()) {   // X1 = dO' A^T
            ok = mbar_wait(&bars[2], ph);
            if (ok) pend &= ~0x4u;
            if (ok) {
                tc_fence_after();
    #pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16(taddr + X1, kmajor_desc(u3, 128, k), kmajor_desc(uA, 128, k), id_kk, k > 0);
                bulk_wait_read_all();   // the dv store has read T_S before the P3 epilogue rewrites it
                mma_commit(&bars[4]);
            }
        }
        wait_mma();
        if (issuer() && it + 1 < i1) issue_v(it + 1, T_A);   // A is consumed: the next item's V
        {   // P3 = s (dO' A^T) o Gamma (the s of q~ = s q folded in, exactly as bwd_chunk1_tc does)
            float x[32];
            tmem_ld16x2(tl + X1, x);
            mask_scores(x, scale);
            store_q<__half>(T_S, row, c0, x);
            if (ok) ok = mbar_wait(&bars[3], ph) && mbar_wait(&bars[1], ph);
            if (tid == 0 && ok) pend &= ~0xAu;
            if (ok) {   // Q and K: bf16 -> fp16
                bf16_to_f16_q(L1, row, c0);
                bf16_to_f16_q(L2, row, c0);
            }
        }
        publish();
        if (issuer()) {   // X2 = P3^T Q (intra part of dk) ;  X1 = Q K^T
    #pragma unroll
            for (int k = 0; k < 8; ++k) {
                mma_bf16(taddr + X2, mnmajor_desc(uS, 128, k), mnmajor_desc(u1, 128, k), id_nn, k > 0);
                mma_bf16(taddr + X1, kmajor_desc(u1, 128, k), kmajor_desc(u2, 128, k), id_kk, k > 0);
            }
            mma_commit(&bars[4]);
        }
        wait_mma();
        if (issuer() && it + 1 < i1) issue_do(it + 1, L1);   // Q is consumed: the next item's dO
        {   // <k, (P3^T Q)_t> ; P1 = s (Q K^T) o Gamma ; K -> K->
            float x[32], kv[32];
            tmem_ld16x2(tl + X2, x);
            load_q(L2, row, c0, kv);
            cG += dot32(kv, x);
            tmem_ld16x2(tl + X1, x);
            mask_scores(x, scale);
            store_q<__half>(T_S, row, c0, x);
            __syncthreads();   // the Q K^T product has read K; rows are rescaled in place below
            if (ok) scale_q(L2, row, c0, fw);
        }
        publish();
        if (issuer()) {   // X1 = A-> D^K (inter part of dk) ; X3 += P1^T dO' ; X4 += K-> D^K^T
    #pragma unroll
            for (int k = 0; k < 8; ++k) {
                mma_bf16(taddr + X1, kmajor_desc(uAS, 128, k), mnmajor_desc(u4, 128, k), id_kn, k > 0);
                mma_bf16(taddr + X3, mnmajor_desc(uS, 128, k), mnmajor_desc(u3, 128, k), id_nn, 1u);
                mma_bf16(taddr + X4, kmajor_desc(u2, 128, k), kmajor_desc(u4, 128, k), id_kk, 1u);
            }
            mma_commit(&bars[4]);
        }
        wait_mma();
        if (issuer() && it + 1 < i1) issue_first(it + 1, L3, L4);   // the next item's O'', D^V
        float cIG = 0.f, cL = 0.f, cIL = 0.f, db = 0.f;
        if (ok) {
            float x[32], y[32];
            tmem_ld16x2_pair(tl + X2, x, tl + X1, y);   // dk = P3^T Q + A-> D^K
    #pragma unroll
            for (int i = 0; i < 32; ++i) x[i] += y[i];
            store_q<__nv_bfloat16>(T_S, row, c0, x);   // dk, staged (P1 is consumed) for a TMA store
            float av[32];
            write_vector_q_vals(av, hf, u, lam, beta, sl);   // unrounded a
            tmem_ld16x2_pair(tl + X3, x, tl + X4, y);   // intra- / inter-chunk da (both passes)
    #pragma unroll
            for (int i = 0; i < 32; ++i) db = fmaf(x[i] + y[i], av[i], db);
    #pragma unroll
            for (int i = 0; i < 32; ++i) av[i] = round16<__half>(av[i]);   // a as the MMAs saw it
            cL = -omega_dot_q(x, av, hf, u, sl);
            cIG = dot32(av, y);
            cIL = -omega_dot_q(y, av, hf, u, sl);
        }
        // row sums over the four column quarters, staged in the scaled write-vector tile (its last
        // product is complete; the next item rewrites it after its first barrier)
        float* s_fin = reinterpret_cast<float*>(T_AS);   // [5][4][128]
        fence_async_smem();   // the staged dk rows, for the TMA store after the barrier below
        s_fin[(0 * 4 + cq) * 128 + row] = cG;
        s_fin[(1 * 4 + cq) * 128 + row] = cL;
        s_fin[(2 * 4 + cq) * 128 + row] = db;
        s_fin[(3 * 4 + cq) * 128 + row] = cIG;
        s_fin[(4 * 4 + cq) * 128 + row] = cIL;
        ok = __syncthreads_and(ok);
        if (issuer()) {
            tma_store_3d(&tdk, T_S, 0, h, rowtok);
            tma_store_3d(&tdk, T_S + TILE / 2, 64, h, rowtok);
            bulk_commit();
        }
        if (cq == 0 && ok) {
            float v[5];
    #pragma unroll
            for (int k = 0; k < 5; ++k) {
                const float* r = s_fin + 4 * 128 * k + row;
                v[k] = (r[0] + r[128]) + (r[256] + r[384]);
            }
            const size_t BTH = (size_t)s.B * s.T * s.H;
            a.tok[2 * BTH + gi] = v[0];
            a.tok[3 * BTH + gi] = v[1];
            a.tok[4 * BTH + gi] = v[2] / beta;
            a.tok[5 * BTH + gi] = v[3];
            a.tok[6 * BTH + gi] = v[4];
        }
        ph ^= 1;
        {
            const int t = rA;
            rA = rL2;
            rL2 = t;
        }
    }
    ok = __syncthreads_and(ok);
    if (!ok && tid == 0) {
        flag_error(CYFA_ERR_TIMEOUT);
        // let copies still in flight land before the shared memory is released
        for (int k = 0; k < 7; ++k)
            if (pend & (1u << k)) mbar_wait(&bars[k], (pend >> (8 + k)) & 1);
    }
    if (tid == 0) bulk_wait_all();
    tc_fence_before();
    __syncthreads();
    if (ro.warp == 0) tmem_dealloc(taddr, 512);
}

// ---------------------------------------------------------------------------------------
// dR (Sec. 3.3: the middle readout l = M z, p = softmax(l), y = M^T p with M = R Phi): the
// gradient of M is dM = sum_t (dl_t z_t^T + p_t dy_t^T), summed over the batch; then
// dR = dM Phi^T.  dm_reduce_tc: CTA (h, split) runs over its share of the head's 128-token
// chunks (all batch rows) and accumulates DL^T Z + P^T DY on tcgen05 in TMEM (the vectors were
// written in fp16 by bwd_chunk1_tc), streaming pairs of tiles through a three-stage TMA ring.
constexpr int DM_NS = 3;

__global__ void __launch_bounds__(256, 1) dm_reduce_tc(const __grid_constant__ CUtensorMap tz,
                                                        const __grid_constant__ CUtensorMap tp,
                                                        const __grid_constant__ CUtensorMap tdy,
                                                        const __grid_constant__ CUtensorMap tdl,
                                                        TcBwdArgs a) {
    const Shape s = a.s;
    const int h = blockIdx.x, split = blockIdx.y;
    const int nct = s.T / CT, nch = s.B * nct;   // the head's chunks over the batch
    const int c0i = (int)((long long)nch * split / a.dm_split);
    const int c1i = (int)((long long)nch * (split + 1) / a.dm_split);
    const int NT = 2 * (c1i - c0i);              // steps: (DL, Z) then (P, DY) per chunk
    const int tid = threadIdx.x, warp = tid >> 5;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    uint64_t* bar_tma = reinterpret_cast<uint64_t*>(smem);
    uint64_t* bar_mma = bar_tma + DM_NS;
    uint32_t* s_taddr = reinterpret_cast<uint32_t*>(smem + 128);
    uint8_t* tiles = smem + 1024;   // [stage][X | Y]
    if (tid == 0) {
        for (int i = 0; i < 2 * DM_NS; ++i) mbar_init(&bar_tma[i], 1);
        fence_mbar_init();
    }
    if (warp == 0) tmem_alloc(s_taddr, 128);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *s_taddr;
    int issued = 0, landed = 0;
    auto issue = [&](int it) {
        const int st = it % DM_NS, ch = c0i + it / 2, b = ch / nct, c = ch - b * nct;
        const int rowbh = (b * s.H + h) * s.T + c * CT;
        uint8_t* tX = tiles + (2 * st) * TILE;
        const CUtensorMap* mx = (it & 1) ? &tp : &tdl;
        const CUtensorMap* my = (it & 1) ? &tdy : &tz;
        mbar_expect_tx(&bar_tma[st], 2 * TILE);
        tma_load_2d(tX, mx, 0, rowbh, &bar_tma[st]);
        tma_load_2d(tX + TILE / 2, mx, 64, rowbh, &bar_tma[st]);
        tma_load_2d(tX + TILE, my, 0, rowbh, &bar_tma[st]);
        tma_load_2d(tX + TILE + TILE / 2, my, 64, rowbh, &bar_tma[st]);
        ++issued;
    };
    if (tid == 0)
        for (int i = 0; i < DM_NS - 1 && i < NT; ++i) issue(i);
    bool ok = true;
    const uint32_t id_nn = idesc_f16(128, 128, 1, 1);
    if (tid == 0) {   // one thread runs the ring: the tiles need no touch-up
        for (int it = 0; it < NT && ok; ++it) {
            const int st = it % DM_NS;
            if (it >= 1) ok = mbar_wait(&bar_mma[(it - 1) % DM_NS], ((it - 1) / DM_NS) & 1);
            if (ok && it + DM_NS - 1 < NT) issue(it + DM_NS - 1);
            if (ok) ok = mbar_wait(&bar_tma[st], (it / DM_NS) & 1);
            if (!ok) break;
            ++landed;
            tc_fence_after();
            const uint32_t uX = smem_u32(tiles + (2 * st) * TILE), uY = uX + TILE;
#pragma unroll
            for (int k = 0; k < 8; ++k)
                mma_bf16(taddr, mnmajor_desc(uX, 128, k), mnmajor_desc(uY, 128, k), id_nn,
                         (it == 0 && k == 0) ? 0u : 1u);
            mma_commit(&bar_mma[st]);
        }
        if (ok && NT > 0) ok = mbar_wait(&bar_mma[(NT - 1) % DM_NS], ((NT - 1) / DM_NS) & 1);
    }
    tc_fence_after();
    ok = __syncthreads_and(ok);
    float* dst = a.dMp + ((size_t)h * a.dm_split + split) * 128 * 128;
    const int q = warp & 3, hf = warp >> 2, lrow = 32 * q + (tid & 31);
    if (ok && NT > 0) {
        float x[64];
        tmem_ld64(taddr + ((uint32_t)(32 * q) << 16) + 64 * hf, x);
#pragma unroll
        for (int i = 0; i < 64; i += 4)
            *reinterpret_cast<float4*>(dst + lrow * 128 + 64 * hf + i) = make_float4(x[i], x[i + 1], x[i + 2], x[i + 3]);
    } else if (ok) {   // no chunk in this split
        for (int i = 0; i < 64; ++i) dst[lrow * 128 + 64 * hf + i] = 0.f;
    } else if (tid == 0) {
        flag_error(CYFA_ERR_TIMEOUT);
        for (int i = landed; i < issued; ++i) mbar_wait(&bar_tma[i % DM_NS], (i / DM_NS) & 1);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(taddr, 128);
}

// dR[h][i][k] = sum_j dM[h][i][j] Phi[k][j] for the m active slots i, k (dM summed over the
// splits; its column j in the kernels' Fourier order when tc_order, else in the paper's).  One
// block per (h, i).
__global__ void __launch_bounds__(128) dr_finalize_kernel(const float* dMp, int dm_split,
                                                          bool tc_order, float* dR, Slots sl) {
    const int h = blockIdx.x, i = blockIdx.y, t = threadIdx.x;
    const int m = sl.m;
    __shared__ float s_dm[128], s_ct[MA], s_st[MA];
    {
        float acc = 0.f;
        const float* src = dMp + (size_t)h * dm_split * 128 * 128 + i * 128 + t;
        for (int sp = 0; sp < dm_split; ++sp) acc += src[(size_t)sp * 128 * 128];
        s_dm[tc_order ? paper_slot(t) : t] = acc;   // paper order: DC, cos_1, sin_1, ..., pad
    }
    if (t < m) {
        float sv, cv;
        sincospif((float)t * sl.two_over_m, &sv, &cv);
        s_ct[t] = cv;
        s_st[t] = sv;
    }
    __syncthreads();
    if (t < m) {   // k = t: Phi[k][0] = 1/sqrt(m), Phi[k][2j-1] = sqrt(2/m) cos(2 pi j k / m), ...
        float acc = s_dm[0] * sl.inv_sqrt_m;
        float ac = 0.f, as = 0.f;
        int idx = 0;
        for (int j = 1; j <= sl.npair; ++j) {
            idx += t;
            if (idx >= m) idx -= m;
            ac = fmaf(s_dm[2 * j - 1], s_ct[idx], ac);
            as = fmaf(s_dm[2 * j], s_st[idx], as);
        }
        dR[((size_t)h * m + i) * m + t] = acc + sl.sqrt2_over_m * (ac + as);
    }
}

// Gate gradients of one chunk: chunk-local suffix sums of the per-token scalars plus the
// state-level term of everything after the chunk, then the activation derivatives.
__global__ void __launch_bounds__(128) tc_gate_kernel(TcBwdArgs a) {
    const Shape s = a.s;
    const int bh = blockIdx.x, cg = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nct = s.T / CT, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const size_t BTH = (size_t)s.B * s.T * s.H;
    const size_t gi = ((size_t)b * s.T + cg * CT + tid) * s.H + h;
    // row side (bwd_chunk1_tc) minus intra-chunk column side (bwd_chunk2_tc): suffix sums;
    // inter-chunk column side: prefix sums over the earlier tokens of the chunk
    const float xg = a.tok[gi] - a.tok[2 * BTH + gi];
    const float xl = a.tok[BTH + gi] + a.tok[3 * BTH + gi];
    const float pg = a.tok[5 * BTH + gi];
    const float pl = a.tok[6 * BTH + gi];
    float sg = xg, sl = xl;   // inclusive suffix
    float qg = pg, ql = pl;   // inclusive prefix
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float yg = __shfl_down_sync(0xffffffffu, sg, o);
        const float yl = __shfl_down_sync(0xffffffffu, sl, o);
        const float ug = __shfl_up_sync(0xffffffffu, qg, o);
        const float ul = __shfl_up_sync(0xffffffffu, ql, o);
        if (lane + o < 32) {
            sg += yg;
            sl += yl;
        }
        if (lane >= o) {
            qg += ug;
            ql += ul;
        }
    }
    __shared__ float s_w[4][4];
    __shared__ double s_dA[4];
    if (lane == 0) {
        s_w[0][warp] = sg;
        s_w[1][warp] = sl;
    }
    if (lane == 31) {
        s_w[2][warp] = qg;
        s_w[3][warp] = ql;
    }
    __syncthreads();
    for (int w = warp + 1; w < 4; ++w) {
        sg += s_w[0][w];
        sl += s_w[1][w];
    }
    for (int w = 0; w < warp; ++w) {
        qg += s_w[2][w];
        ql += s_w[3][w];
    }
    qg -= pg;   // exclusive prefix: tokens before this one
    ql -= pl;
    const float* bd = a.bnd + ((size_t)bh * nct + cg) * 2;
    const float dlogalpha = sg + qg + bd[0];
    const float ddelta = sl - ql + bd[1];
    const float f = a.decay_logit[gi];
    a.d_decay[gi] = dlogalpha * (-a.A[h] * sigmoidf_(f));
    if (a.d_clock) {   // no clock logits (fixed-rate clock): no clock gradient
        const float delta = sigmoidf_(a.clock_logit[gi]);
        a.d_clock[gi] = ddelta * delta * (1.f - delta);
    }
    const float bt = a.beta[gi];
    const float dbeta = a.tok[4 * BTH + gi];
    a.d_beta[gi] = dbeta * bt * (1.f - bt);
    // every per-token intermediate of the backward (fp16 snapshots, adjoints, o'', dL/do')
    // feeds these three sums, so an fp16 overflow anywhere reaches them as inf / NaN
    if (!isfinite(dlogalpha + ddelta + dbeta)) flag_error(CYFA_ERR_RANGE);
    double da = (double)dlogalpha * (double)(-softplusf_(f));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) da += __shfl_xor_sync(0xffffffffu, da, o);
    if (lane == 0) s_dA[warp] = da;
    __syncthreads();
    if (tid == 0) a.dA_part[(size_t)bh * nct + cg] = s_dA[0] + s_dA[1] + s_dA[2] + s_dA[3];
}

// dA[h] = sum over batch rows and chunks of the per-chunk partials; one block per head.
__global__ void __launch_bounds__(256) tc_dA_kernel(TcBwdArgs a) {
    const int h = blockIdx.x, tid = threadIdx.x;
    const int nct = a.s.T / CT, n = a.s.B * nct;
    double t = 0.0;
    for (int i = tid; i < n; i += 256) {
        const int b = i / nct, c = i - b * nct;
        t += a.dA_part[((size_t)b * a.s.H + h) * nct + c];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    __shared__ double s_t[8];
    if ((tid & 31) == 0) s_t[tid >> 5] = t;
    __syncthreads();
    if (tid == 0) {
        double r = 0.0;
        for (int w = 0; w < 8; ++w) r += s_t[w];
        a.dA[h] = (float)r;
    }
}

}  // namespace

template <class SL>
cudaError_t launch_bwd_tc_sl(const TcBwdArgs& a, const TcFwdArgs& f, const void* q, const void* k,
                             const void* v, const void* dO, cudaStream_t st) {
    const Shape& s = a.s;
    const int nct = s.T / CT;
    const unsigned long long BH = (unsigned long long)s.B * s.H;
    CUtensorMap mq, mk, mv, mdo, mm, msf, msa, mo2, mdo1, mdq;
    if (!tc_qkv_maps(s, q, k, v, &mq, &mk, &mv) || !tc_qkv_maps(s, dO, nullptr, nullptr, &mdo, nullptr, nullptr) ||
        !tc_qkv_maps(s, a.dq, nullptr, nullptr, &mdq, nullptr, nullptr) ||
        !tc_rows_map(&mm, a.Mb, (unsigned long long)s.H * 128, true) ||
        !tc_rows_map(&msf, a.snapF, BH * nct * 2 * 128, true) ||
        !tc_rows_map(&msa, a.snapA, BH * nct * 2 * 128, true) ||
        !tc_rows_map(&mo2, a.O2, BH * s.T, true) || !tc_rows_map(&mdo1, a.DO1, BH * s.T, true))
        return cudaErrorInvalidValue;
    // chunk-start states: the forward's saved snapshots, or recomputed (segment states, then a
    // walk of every segment)
    cudaError_t e = a.saved ? launch_segment_decay(f, st) : launch_fwd_segment_states(f, k, v, st);
    if (e != cudaSuccess) return e;
    // heads fastest: the CTAs that read the same token rows of q, k, v, dO run together
    const dim3 gseg(s.B * s.H, a.nseg), gchunk(s.B * s.H, nct);
    const int sm_walk6 = 1024 + 6 * TILE + 1024;
    const int sm_snap_adj = 1024 + 4 * TC_SEGC * CT + 6 * TILE + 1024;
    const int sm_adj_seg = 1024 + 4 * TC_SEGC * CT + 6 * TILE + 1024;
    const int sm_chunk1 = 8192 + 6 * TILE + 1024, sm_chunk2 = 2048 + 7 * TILE + 1024;
    if (!a.saved) {
        cudaFuncSetAttribute(snap_fwd_tc<SL>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm_walk6);
        { LaunchScope ls_("tc_snap_fwd", st); snap_fwd_tc<SL><<<gseg, 256, sm_walk6, st>>>(mk, mv, a); }
    }
    cudaFuncSetAttribute(bwd_chunk1_tc<SL>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm_chunk1);
    {   // persistent: one CTA per SM walks a contiguous range of (b*h, chunk) items
        int dev = 0, sms = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            return cudaErrorInvalidValue;
        const long long items = (long long)s.B * s.H * nct;
        const int grid1 = (int)(items < sms ? items : sms);
        // the staged vectors of dR go out by TMA store; without dR the maps are unused stand-ins
        CUtensorMap mz, mpp, mdy, mdl;
        const void* bz = a.mZ ? (const void*)a.mZ : (const void*)a.DO1;
        const void* bp = a.mP ? (const void*)a.mP : (const void*)a.DO1;
        const void* bdy = a.mDY ? (const void*)a.mDY : (const void*)a.DO1;
        const void* bdl = a.mDL ? (const void*)a.mDL : (const void*)a.DO1;
        if (!tc_rows_map(&mz, bz, BH * s.T, true) || !tc_rows_map(&mpp, bp, BH * s.T, true) ||
            !tc_rows_map(&mdy, bdy, BH * s.T, true) || !tc_rows_map(&mdl, bdl, BH * s.T, true))
            return cudaErrorInvalidValue;
        LaunchScope ls_("tc_bwd_chunk1", st);
        bwd_chunk1_tc<SL><<<grid1, 512, sm_chunk1, st>>>(mq, mk, mv, mdo, mm, msf, mz, mpp, mdy, mdl, mdq, a);
    }
    cudaFuncSetAttribute(adj_walk_tc<false, SL>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm_adj_seg);
    { LaunchScope ls_("tc_adj_segment", st); adj_walk_tc<false, SL><<<gseg, 256, sm_adj_seg, st>>>(mdo1, mo2, mq, mdo, msf, msa, a); }
    { LaunchScope ls_("tc_adj_scan", st); seg_scan_rev_kernel<<<dim3(128, s.B * s.H), 256, 0, st>>>(a); }
    cudaFuncSetAttribute(adj_walk_tc<true, SL>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm_snap_adj);
    { LaunchScope ls_("tc_snap_adj", st); adj_walk_tc<true, SL><<<gseg, 256, sm_snap_adj, st>>>(mdo1, mo2, mq, mdo, msf, msa, a); }
    cudaFuncSetAttribute(bwd_chunk2_tc<SL>, cudaFuncAttributeMaxDynamicSharedMemorySize, sm_chunk2);
    {
        int dev = 0, sms = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            return cudaErrorInvalidValue;
        const long long items = (long long)s.B * s.H * nct;
        const int grid2 = (int)(items < sms ? items : sms);
        LaunchScope ls_("tc_bwd_chunk2", st);
        CUtensorMap mdk, mdv;
        if (!tc_qkv_maps(s, a.dk, a.dv, nullptr, &mdk, &mdv, nullptr)) return cudaErrorInvalidValue;
        bwd_chunk2_tc<SL><<<grid2, 512, sm_chunk2, st>>>(mq, mk, mv, mdo, mo2, mdo1, msa, mdk, mdv, a);
    }
    { LaunchScope ls_("tc_gate", st); tc_gate_kernel<<<gchunk, 128, 0, st>>>(a); }
    if (a.dR) {   // dR from the middle-readout vectors bwd_chunk1_tc wrote
        CUtensorMap mz, mp, mdy, mdl;
        if (!tc_rows_map(&mz, a.mZ, BH * s.T, true) || !tc_rows_map(&mp, a.mP, BH * s.T, true) ||
            !tc_rows_map(&mdy, a.mDY, BH * s.T, true) || !tc_rows_map(&mdl, a.mDL, BH * s.T, true))
            return cudaErrorInvalidValue;
        const int sm_dm = 1024 + 2 * DM_NS * TILE + 1024;
        cudaFuncSetAttribute(dm_reduce_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, sm_dm);
        { LaunchScope ls_("tc_dm_reduce", st); dm_reduce_tc<<<dim3(s.H, a.dm_split), 256, sm_dm, st>>>(mz, mp, mdy, mdl, a); }
        e = launch_dr_finalize(a.dMp, a.dm_split, s.H, true, a.dR, s.sl, st);
        if (e != cudaSuccess) return e;
    }
    if (a.dA) { LaunchScope ls_("tc_dA", st); tc_dA_kernel<<<s.H, 256, 0, st>>>(a); }
    return cudaGetLastError();
}

cudaError_t launch_bwd_tc(const TcBwdArgs& a, const TcFwdArgs& f, const void* q, const void* k,
                          const void* v, const void* dO, cudaStream_t st) {
    return a.s.sl.m == 127 ? launch_bwd_tc_sl<Slots127>(a, f, q, k, v, dO, st)
                           : launch_bwd_tc_sl<Slots>(a, f, q, k, v, dO, st);
}

cudaError_t launch_dr_finalize(const float* dMp, int dm_split, int H, bool tc_order, float* dR,
                               const Slots& sl, cudaStream_t st) {
    { LaunchScope ls_("dr_finalize", st); dr_finalize_kernel<<<dim3(H, sl.m), 128, 0, st>>>(dMp, dm_split, tc_order, dR, sl); }
    return cudaGetLastError();
}

cudaError_t tc_bwd_read_error(cudaStream_t st, int* err) {
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
