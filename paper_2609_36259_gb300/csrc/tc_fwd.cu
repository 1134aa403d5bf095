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
#include "tc_chunk.cuh"

namespace cyfa {

namespace {

using namespace tc;

// ---------------------------------------------------------------------------------------
template <int SEGC, typename OT, class SL>
__global__ void __launch_bounds__(512, 1) seg_state_tc(const __grid_constant__ CUtensorMap tk,
                                                        const __grid_constant__ CUtensorMap tv,
                                                        TcFwdArgs a) {
    const Shape s = a.s;
    const SL sl = slots_of<SL>(s);
    const int bh = blockIdx.x, seg = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nct = s.T / CT;
    const int c_begin = seg * SEGC;
    const int nc = min(SEGC, nct - c_begin);
    const int tid = threadIdx.x;
    const QRole ro;   // 512 threads: one row and one column quarter each
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem);              // tma[2], mma[2]
    uint32_t* s_taddr = reinterpret_cast<uint32_t*>(smem + 64);
    float* s_tot = reinterpret_cast<float*>(smem + 128);             // [SEGC]
    float* s_sfx = s_tot + SEGC;                                     // [SEGC]
    float* s_lam = reinterpret_cast<float*>(smem + 1024);            // [SEGC * CT] per token
    float* s_beta = s_lam + SEGC * CT;
    float* s_gs = s_beta + SEGC * CT;                                // chunk-local decays
    uint8_t* tiles = smem + 1024 + 12 * SEGC * CT;                   // [buf][A | K | V]
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
    if (tid == 0) {   // chunk 0's K and V are on their way while the gates load
        for (int i = 0; i < 4; ++i) mbar_init(&bars[i], 1);
        fence_mbar_init();
        issue_kv(0, 0);
    }
    {   // every token's gates, loaded once: all of a thread's loads in flight together
        constexpr int NPT = SEGC * CT / 512;
        float l[NPT], be[NPT], v[NPT], w[NPT];
#pragma unroll
        for (int k = 0; k < NPT; ++k) {
            const int i = tid + 512 * k;
            const int t0 = (c_begin + i / CT) * CT, t = t0 + i % CT;
            const size_t gi = ((size_t)b * s.T + t) * s.H + h;
            const bool in = i < nc * CT;
            l[k] = in ? a.lam[gi] : 0.f;
            be[k] = in ? a.beta[gi] : 0.f;
            v[k] = in ? a.g[gi] : 0.f;
            w[k] = (in && s.Cg == 64 && t - t0 >= 64) ? a.g[((size_t)b * s.T + t0 + 63) * s.H + h] : 0.f;
        }
#pragma unroll
        for (int k = 0; k < NPT; ++k) {
            const int i = tid + 512 * k;
            if (i < nc * CT) {
                s_lam[i] = l[k];
                s_beta[i] = be[k];
                s_gs[i] = v[k] + w[k];   // cum128
            }
        }
    }

    if (ro.warp == 0) tmem_alloc(s_taddr, 256);
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
    __syncthreads();
    bool ok = true;
    constexpr bool F16 = std::is_same<OT, __half>::value;
    // one N = 256 product per K-step: B = [K | V] (adjacent tiles, 64-column blocks 16 KiB apart),
    // D = [Kbar | Vbar] (TMEM columns 0 .. 255), the A-> operand read once
    const uint32_t idesc = idesc_k16<OT>(128, 256, 1, 1);
    for (int c = 0; c < nc; ++c) {
        const int buf = c & 1;
        // A-> rows of this chunk, scaled by the decay from the token to the segment end (its
        // buffer's last reader, product c - 2, is complete; product c - 1 runs meanwhile)
        {
            const int i = c * CT + ro.row;
            const float w = s_beta[i] * ex2((s_tot[c] - s_gs[i] + s_sfx[c]) * LOG2E);
            write_vector_q<OT>(tiles + 3 * buf * TILE, ro.row, ro.hf, ro.u, s_lam[i], w, sl);
        }
        if (c >= 1 && ok) ok = mbar_wait(&bars[2 + ((c - 1) & 1)], ((c - 1) >> 1) & 1);
        if (tid == 0 && ok && c + 1 < nc) issue_kv(c + 1, (c + 1) & 1);
        if (tid == 0 && c + 2 < nc) {   // the chunk after into L2: its load then comes from there
            const int r2 = b * s.T + (c_begin + c + 2) * CT;
            tma_prefetch_3d(&tk, 0, h, r2);
            tma_prefetch_3d(&tk, 64, h, r2);
            tma_prefetch_3d(&tv, 0, h, r2);
            tma_prefetch_3d(&tv, 64, h, r2);
        }
        if (F16) {   // the bf16 K and V tiles become fp16 operands
            if (ok) ok = mbar_wait(&bars[buf], (c >> 1) & 1);
            if (ok) {
                bf16_to_f16_q(tiles + (3 * buf + 1) * TILE, ro.row, ro.c0);
                bf16_to_f16_q(tiles + (3 * buf + 2) * TILE, ro.row, ro.c0);
            }
        }
        fence_async_smem();
        ok = __syncthreads_and(ok);
        if (!ok) break;
        if (tid == 0) {
            if (F16 || mbar_wait(&bars[buf], (c >> 1) & 1)) {
                tc_fence_after();
                const uint32_t tA = smem_u32(tiles + 3 * buf * TILE);
                const uint32_t tK = smem_u32(tiles + (3 * buf + 1) * TILE);
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16(taddr, mnmajor_desc(tA, 128, k), mnmajor_desc(tK, 128, k), idesc,
                             (c > 0 || k > 0) ? 1u : 0u);
                mma_commit(&bars[2 + buf]);
            }
        }
    }
    if (ok) ok = mbar_wait(&bars[2 + ((nc - 1) & 1)], ((nc - 1) >> 1) & 1);
    tc_fence_after();
    ok = __syncthreads_and(ok);
    if (ok) {   // [Kbar | Vbar] delta out through the (now idle) tiles, coalesced
        float* stage = reinterpret_cast<float*>(tiles);
        const uint32_t tl = taddr + ((uint32_t)(32 * ro.q) << 16) + 64 * ro.cq;
        for (int c0 = 0; c0 < 64; c0 += 32) {
            float v[32];
            tmem_ld32(tl + c0, v);
#pragma unroll
            for (int i = 0; i < 32; i += 4)
                *reinterpret_cast<float4*>(stage + ro.row * STAGE_LD + 64 * ro.cq + c0 + i) =
                    make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
        }
        __syncthreads();
        stage_to_global_128x256(a.segS + ((size_t)bh * a.nseg + seg) * 128 * 256, stage, tid, 512);
    } else if (tid == 0) {
        flag_error(CYFA_ERR_TIMEOUT);
        // let copies still in flight land before the shared memory is released
        for (int i = 0; i < 2; ++i) mbar_wait(&bars[i], 0);
    }
    tc_fence_before();
    __syncthreads();
    if (ro.warp == 0) tmem_dealloc(taddr, 256);
}

// Segment-start states: S_start(0) = initial state, S_start(j+1) = exp(G_j) S_start(j) + dS(j),
// in place over the dS buffer (tensor-core row order); the final state goes to Kout / Vout in
// the paper's row order.  Up to 32 segments are loaded before they are folded in.
__global__ void __launch_bounds__(256) seg_scan_kernel(TcFwdArgs a) {
    const int bh = blockIdx.y;
    const int e = blockIdx.x * 256 + threadIdx.x;   // element of the [128 x 256] state block
    const int row = e >> 8, col = e & 255;
    const bool isK = col < 128;
    const int dcol = col & 127;
    const int prow = paper_slot(row);
    float S = 0.f;
    const float* init = isK ? a.Kbar0 : a.Vbar0;
    if (init) S = init[((size_t)bh * 128 + prow) * 128 + dcol];
    float* base = a.segS + (size_t)bh * a.nseg * 128 * 256 + e;
    const float* G = a.segG + (size_t)bh * a.nseg;
    for (int j0 = 0; j0 < a.nseg; j0 += 32) {
        float d[32], gj[32];   // all loads first: the stores below may alias them
#pragma unroll
        for (int u = 0; u < 32; ++u) {
            const bool in = j0 + u < a.nseg;
            d[u] = in ? base[(size_t)(j0 + u) * 128 * 256] : 0.f;
            gj[u] = in ? G[j0 + u] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 32; ++u) {
            if (j0 + u < a.nseg) {
                base[(size_t)(j0 + u) * 128 * 256] = S;
                S = expf(gj[u]) * S + d[u];
            }
        }
    }
    float* out = isK ? a.Kout : a.Vout;
    if (out) out[((size_t)bh * 128 + prow) * 128 + dcol] = S;
}

// ---------------------------------------------------------------------------------------
// Chunk walk of one (b, h, segment), warp-specialised.  640 threads in two groups:
//  * chain (warps 0-15, 512 threads): thread (row, quarter) owns TMEM lane `row` and the column
//    quarter of QRole in the two product accumulators X1, X2; it runs the epilogues of the
//    output chain Q K^T, Q Kbar^T -> P1 -> P1 A -> z -> z M^T -> softmax -> p M -> o'' ->
//    O'' A^T, O'' Vbar -> P2 -> P2 V -> o.  Thread 0 issues the chain's MMAs.
//  * state (warps 16-19, 128 threads): thread r owns row r of every tile and TMEM lane r of the
//    state accumulators [Kbar | Vbar]; it builds the write vectors a (T_A) and A-> (T_Q), takes
//    the fp16 state snapshots (T_N), scales the state by gamma^C, converts the bf16 inputs to
//    fp16 and issues the TMA loads, the state-update MMAs and the snapshot stores.  Thread 512
//    leads.
// The state work of chunk c (snapshot of Vbar, A->, scaling, V) runs under the chain's products
// and epilogues; the state update [Kbar | Vbar] += A->^T [K | V] is issued by the state leader as
// soon as its operands are ready, so the chain's commits never wait for it.  The groups meet on
// mbarriers only:
//   F1 / F5 / F6  chain products 1, 5, 6 of the chunk complete (tiles they read are free)
//   SR            state ready: Vbar snapshot in T_N, A-> in T_Q, state scaled, V converted
//   SU            state update (issued by the state leader) complete
//   NX            next chunk's a and Kbar snapshot in place (the chain converts its Q, K)
enum { OB_QK, OB_V, OB_M, OB_MMA, OB_F1, OB_F5, OB_F6, OB_SU, OB_SR, OB_NX, OB_END, OB_ENDS, OB_N };
constexpr int OUT_CHAIN = 512, OUT_THREADS = 640;

// Bounded wait (WAIT_LIMIT_NS) that also gives up once the other group has flagged an abort.
__device__ __forceinline__ bool mbar_wait_ab(uint64_t* bar, uint32_t parity, volatile int* abort_) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort_ || globaltimer_ns() - t0 > WAIT_LIMIT_NS) return false;
    }
}
__device__ __forceinline__ void named_sync(uint32_t id, uint32_t n) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
// Barrier `id` over n threads that also ANDs a predicate across them.
__device__ __forceinline__ bool named_and(uint32_t id, uint32_t n, bool v) {
    uint32_t r;
    asm volatile(
        "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.and.pred q, %2, %3, p;\n"
        " selp.u32 %0, 1, 0, q;\n}\n"
        : "=r"(r)
        : "r"((uint32_t)v), "r"(id), "r"(n)
        : "memory");
    return r != 0;
}

template <int SEGC, class SL>
__global__ void __launch_bounds__(OUT_THREADS, 1) seg_out_tc(const __grid_constant__ CUtensorMap tq,
                                                              const __grid_constant__ CUtensorMap tk,
                                                              const __grid_constant__ CUtensorMap tv,
                                                              const __grid_constant__ CUtensorMap tm,
                                                              const __grid_constant__ CUtensorMap tsnap,
                                                              const __grid_constant__ CUtensorMap to,
                                                              TcFwdArgs a) {
    const Shape s = a.s;
    const SL sl = slots_of<SL>(s);
    const int bh = blockIdx.x, seg = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nct = s.T / CT;
    const int c_begin = seg * SEGC;
    const int nc = min(SEGC, nct - c_begin);
    const int tid = threadIdx.x;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem);          // OB_N mbarriers
    static_assert(OB_N * 8 <= 112, "mbarriers overlap the TMEM address word");
    uint32_t* s_taddr = reinterpret_cast<uint32_t*>(smem + 112);
    volatile int* s_abort = reinterpret_cast<volatile int*>(smem + 116);
    float* s_g2 = reinterpret_cast<float*>(smem + 128);           // [128] log2-domain decays
    float* s_b = s_g2 + 128;                                      // [128] in-block decay factors
    uint8_t* T_Q = smem + 2048;        // Q, then A-> (state-update operand)
    uint8_t* T_K = T_Q + 1 * TILE;
    uint8_t* T_V = T_Q + 2 * TILE;
    uint8_t* T_A = T_Q + 3 * TILE;     // write vectors a_s (rows = tokens)
    uint8_t* T_S = T_Q + 4 * TILE;     // chain staging: P1, z, p, O'', P2 (rows = tokens)
    uint8_t* T_N = T_Q + 5 * TILE;     // state snapshot: Kbar, then Vbar (rows = slots)
    uint8_t* T_M = T_Q + 6 * TILE;     // M = R Phi (rows = slots r, cols = Fourier index)

    if (tid == 0) {
        for (int i = 0; i < OB_N; ++i) mbar_init(&bars[i], 1);
        *s_abort = 0;
        fence_mbar_init();
    }
    if (tid < 32) tmem_alloc(s_taddr, 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t taddr = *s_taddr;
    const uint32_t SK = 0, SV = 128, X1 = 256, X2 = 384;
    const bool save = a.snap != nullptr;
    const uint32_t uQ = smem_u32(T_Q), uK = smem_u32(T_K), uV = smem_u32(T_V),
                   uA = smem_u32(T_A), uS = smem_u32(T_S), uN = smem_u32(T_N),
                   uM = smem_u32(T_M);
    // the snapshot in T_N (part 0: Kbar, 1: Vbar) of chunk cg leaves by a TMA store
    auto store_snap = [&](int cg, int part) {
        const int r = ((bh * nct + cg) * 2 + part) * 128;
        tma_store_2d(&tsnap, T_N, 0, r);
        tma_store_2d(&tsnap, T_N + TILE / 2, 64, r);
        bulk_commit();
    };
    bool ok = true;

    if (tid >= OUT_CHAIN) {
        // ================================================================ state group
        const int r = tid - OUT_CHAIN;                 // row of every tile / TMEM lane
        const uint32_t tlane = taddr + ((uint32_t)(32 * ((tid >> 5) & 3)) << 16);
        const bool leader = tid == OUT_CHAIN;
        const uint32_t id_nn2 = idesc_f16(128, 256, 1, 1);
        static_assert(SV == SK + 128, "the state update writes [Kbar | Vbar] as one accumulator");
        bool su_issued = false;   // leader: a state update that nobody has waited for
        bool qk_pending = false, v_pending = false;
        uint32_t qk_par = 0, v_par = 0;   // parity of the pending loads' phases
        auto issue_qk = [&](int c) {
            const int r0 = b * s.T + (c_begin + c) * CT;
            mbar_expect_tx(&bars[OB_QK], 2 * TILE);
            tma_load_3d(T_Q, &tq, 0, h, r0, &bars[OB_QK]);
            tma_load_3d(T_Q + TILE / 2, &tq, 64, h, r0, &bars[OB_QK]);
            tma_load_3d(T_K, &tk, 0, h, r0, &bars[OB_QK]);
            tma_load_3d(T_K + TILE / 2, &tk, 64, h, r0, &bars[OB_QK]);
            qk_pending = true;
            qk_par = c & 1;
        };
        auto issue_v = [&](int c) {
            const int r0 = b * s.T + (c_begin + c) * CT;
            mbar_expect_tx(&bars[OB_V], TILE);
            tma_load_3d(T_V, &tv, 0, h, r0, &bars[OB_V]);
            tma_load_3d(T_V + TILE / 2, &tv, 64, h, r0, &bars[OB_V]);
            v_pending = true;
            v_par = c & 1;
        };
        // gates of this row's token in chunk c: clock, write strength, log2 decay from the chunk
        // start, and the log2 decay of the whole chunk
        auto gates = [&](int c, float& lam_, float& beta_, float& g2_, float& g2C_) {
            const int t0 = (c_begin + c) * CT;
            const size_t gi = ((size_t)b * s.T + t0 + r) * s.H + h;
            lam_ = a.lam[gi];
            beta_ = a.beta[gi];
            g2_ = cum128(s, a.g, b, h, t0, t0 + r) * LOG2E;
            g2C_ = cum128(s, a.g, b, h, t0, t0 + CT - 1) * LOG2E;
        };
        if (leader) {
            mbar_expect_tx(&bars[OB_M], TILE);
            tma_load_2d(T_M, &tm, 0, h * 128, &bars[OB_M]);
            tma_load_2d(T_M + TILE / 2, &tm, 64, h * 128, &bars[OB_M]);
            issue_qk(0);
            issue_v(0);
        }
        float lam, beta, g2, g2C;
        gates(0, lam, beta, g2, g2C);
#pragma unroll 1
        for (int qq = 0; qq < 4; ++qq) write_vector_q<__half>(T_A, r, qq >> 1, qq & 1, lam, beta, sl);
        if (ok) ok = mbar_wait(&bars[OB_QK], 0);
        if (leader && ok) qk_pending = false;
        if (ok) {
            bf16_to_f16_half(T_Q, r, 0);
            bf16_to_f16_half(T_Q, r, 1);
            bf16_to_f16_half(T_K, r, 0);
            bf16_to_f16_half(T_K, r, 1);
        }
        // the chain group has put the segment-start state into TMEM and the Kbar snapshot
        // into T_N before this barrier
        fence_async_smem();
        tc_fence_before();
        ok = __syncthreads_and(ok);
        tc_fence_after();
        if (ok && leader) {
            if (save) store_snap(c_begin, 0);
            mbar_arrive(&bars[OB_NX]);
        }
        for (int c = 0; c < nc && ok; ++c) {
            const bool last = c + 1 == nc;
            float n_lam = 0.f, n_beta = 0.f, n_g2 = 0.f, n_g2C = 0.f;
            if (!last) gates(c + 1, n_lam, n_beta, n_g2, n_g2C);
            if (leader && !last) {   // the next chunk's Q, K, V into L2: their loads wait for tiles
                const int r1 = b * s.T + (c_begin + c + 1) * CT;
#pragma unroll
                for (int x = 0; x < 128; x += 64) {
                    tma_prefetch_3d(&tq, x, h, r1);
                    tma_prefetch_3d(&tk, x, h, r1);
                    tma_prefetch_3d(&tv, x, h, r1);
                }
            }
            // S1: product 1 has read Q and the Kbar snapshot
            if (ok) ok = mbar_wait_ab(&bars[OB_F1], c & 1, s_abort);
            if (save && leader) bulk_wait_read_all();   // the Kbar snapshot store has read T_N
            tc_fence_after();
            ok = named_and(2, 128, ok);
            if (!ok) break;
            // S2: Vbar snapshot (before scaling), state scaled by gamma^C, A-> rows
            {
                const float gC = ex2(g2C);
#pragma unroll 1
                for (int qq = 0; qq < 4; ++qq) {   // column quarters c0 = 64 (qq / 2) + 16 (qq % 2)
                    const int cc = 64 * (qq >> 1) + 16 * (qq & 1);
                    uint32_t xv[32], xk[32];
                    tmem_ld16x2_async(tlane + SV + cc, xv);
                    if (!last) tmem_ld16x2_async(tlane + SK + cc, xk);
                    tmem_wait_ld();
                    float x[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) x[i] = __uint_as_float(xv[i]);
                    store_q<__half>(T_N, r, cc, x);
                    if (!last) {   // loads and stores of the quarters overlap; one wait at the end
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            xv[i] = __float_as_uint(x[i] * gC);
                            xk[i] = __float_as_uint(__uint_as_float(xk[i]) * gC);
                        }
                        tmem_st16x2_async(tlane + SV + cc, xv);
                        tmem_st16x2_async(tlane + SK + cc, xk);
                    }
                }
                if (!last) {
                    tmem_wait_st();
                    // A-> rows: the fp16 write vector a of the row (T_A) times beta gamma^C / gamma_r
                    const __half2 w2 = __float2half2_rn(ex2(g2C - g2));
#pragma unroll 4
                    for (int j = 0; j < 16; ++j) {
                        const uint32_t off = swz_off(r, 8 * j, 128);
                        uint4 v = *reinterpret_cast<const uint4*>(T_A + off);
                        __half2* e = reinterpret_cast<__half2*>(&v);
#pragma unroll
                        for (int i = 0; i < 4; ++i) e[i] = __hmul2(e[i], w2);
                        *reinterpret_cast<uint4*>(T_Q + off) = v;
                    }
                }
            }
            // S3: V of this chunk
            if (ok) ok = mbar_wait_ab(&bars[OB_V], c & 1, s_abort);
            if (leader && ok) v_pending = false;
            if (ok) {
                bf16_to_f16_half(T_V, r, 0);
                bf16_to_f16_half(T_V, r, 1);
            }
            // S4: publish to the MMA issuer
            fence_async_smem();
            tc_fence_before();
            ok = named_and(2, 128, ok);
            if (!ok) break;
            if (leader) {
                if (save) store_snap(c_begin + c, 1);
                mbar_arrive(&bars[OB_SR]);
                if (!last) {   // state update [Kbar | Vbar] += A->^T [K | V], issued from here so
                               // that the chain's own commits never wait for it; one N = 256
                               // product (T_K, T_V adjacent; SK, SV adjacent)
                    tc_fence_after();
#pragma unroll
                    for (int k = 0; k < 8; ++k)
                        mma_bf16(taddr + SK, mnmajor_desc(uQ, 128, k), mnmajor_desc(uK, 128, k), id_nn2, 1u);
                    mma_commit(&bars[OB_SU]);
                    su_issued = true;
                }
            }
            if (last) break;
            // S5: the state update has read A->, K and V: next Q, K may come in
            if (ok) ok = mbar_wait_ab(&bars[OB_SU], c & 1, s_abort);
            if (ok && leader) {
                su_issued = false;
                issue_qk(c + 1);   // stays pending for the failure path: the chain waits for it
            }
            // S6: product 5 has read a and the Vbar snapshot: next a and the Kbar snapshot
            if (ok) ok = mbar_wait_ab(&bars[OB_F5], c & 1, s_abort);
            if (save && leader) bulk_wait_read_all();   // the Vbar snapshot store has read T_N
            tc_fence_after();
            ok = named_and(2, 128, ok);
            if (!ok) break;
            lam = n_lam;
            beta = n_beta;
            g2 = n_g2;
            g2C = n_g2C;
#pragma unroll 1
            for (int qq = 0; qq < 4; ++qq) {
                const int cc = 64 * (qq >> 1) + 16 * (qq & 1);
                float x[32];
                tmem_ld16x2(tlane + SK + cc, x);
                store_q<__half>(T_N, r, cc, x);
            }
#pragma unroll 1
            for (int qq = 0; qq < 4; ++qq) write_vector_q<__half>(T_A, r, qq >> 1, qq & 1, lam, beta, sl);
            // S8: the next chunk's a and Kbar snapshot are ready (its Q and K are converted to
            // fp16 by the chain group, which is idle at that point)
            fence_async_smem();
            tc_fence_before();
            ok = named_and(2, 128, ok);
            if (!ok) break;
            if (leader) {
                if (save) store_snap(c_begin + c + 1, 0);
                mbar_arrive(&bars[OB_NX]);
            }
            // S9: product 6 has read V: next V may come in
            if (ok) ok = mbar_wait_ab(&bars[OB_F6], c & 1, s_abort);
            if (ok && leader) issue_v(c + 1);
        }
        if (!ok) *s_abort = 1;
        if (leader) {
            if (!ok) {
                flag_error(CYFA_ERR_TIMEOUT);
                if (su_issued) {   // the state update may still be running: let it finish
                    mma_commit(&bars[OB_ENDS]);
                    mbar_wait(&bars[OB_ENDS], 0);
                }
                // copies still in flight land before the shared memory is released
                if (qk_pending) mbar_wait(&bars[OB_QK], qk_par);
                if (v_pending) mbar_wait(&bars[OB_V], v_par);
            }
            if (save) bulk_wait_all();
        }
    } else {
        // ================================================================ chain group
        const QRole ro;
        const int row = ro.row, hf = ro.hf, u = ro.u, c0 = ro.c0, cq = ro.cq;
        const uint32_t tl = taddr + ((uint32_t)(32 * ro.q) << 16) + c0;   // lane, column quarter
        // segment-start state into TMEM; Kbar snapshot into T_N (row = slot)
        {
            const float* src = a.segS + (((size_t)bh * a.nseg + seg) * 128 + row) * 256 + c0;
#pragma unroll
            for (int part = 0; part < 2; ++part) {
                float x[32];
#pragma unroll
                for (int i = 0; i < 32; i += 4) {
                    const float4 f = *reinterpret_cast<const float4*>(src + 128 * part + (i & 15) + 32 * (i >> 4));
                    x[i] = f.x; x[i + 1] = f.y; x[i + 2] = f.z; x[i + 3] = f.w;
                }
                tmem_st16x2(tl + 128 * part, x);
                if (part == 0) store_q<__half>(T_N, row, c0, x);
            }
        }
        fence_async_smem();
        tc_fence_before();
        ok = __syncthreads_and(ok);
        tc_fence_after();
        if (tid == 0 && ok) ok = mbar_wait(&bars[OB_M], 0);
        uint32_t mma_ph = 0;
        const float scale = s.scale;
        const uint32_t id_kk = idesc_f16(128, 128, 0, 0);
        const uint32_t id_kn = idesc_f16(128, 128, 0, 1);
        bool issued = false;   // thread 0: an MMA commit that nobody waited for may be in flight

        auto wait_mma = [&]() {
            if (ok) ok = mbar_wait_ab(&bars[OB_MMA], mma_ph, s_abort);
            mma_ph ^= 1;
            tc_fence_after();
        };
        auto publish = [&]() {
            fence_async_smem();
            tc_fence_before();
            ok = named_and(1, OUT_CHAIN, ok);
            tc_fence_after();
        };
        auto issuer = [&]() { return tid == 0 && ok; };
        auto mask_scores = [&](float (&x)[32], float g2_, float mul) {
            mask_decay_q(x, mul, row, ro.q, c0, g2_, s_g2, s_b);
        };
        // gates of this row's token: prefetched a chunk ahead
        float lam, g2, g2e;
        float n_lam = 0.f, n_ga = 0.f, n_gb = 0.f, n_ge = 0.f;
        auto load_gates = [&](int c, float& l_, float& ga, float& gb, float& ge) {
            const int t0 = (c_begin + c) * CT, t = t0 + row;
            const size_t gi = ((size_t)b * s.T + t) * s.H + h;
            l_ = a.lam[gi];
            // cum128 in two loads: g_cum is local to s.Cg-token chunks (row and row | 15 share
            // the second term)
            ga = a.g[gi];
            gb = (s.Cg == 64 && t - t0 >= 64) ? a.g[((size_t)b * s.T + t0 + 63) * s.H + h] : 0.f;
            ge = a.g[((size_t)b * s.T + t0 + (row | 15)) * s.H + h];
        };
        {
            float ga, gb, ge;
            load_gates(0, lam, ga, gb, ge);
            g2 = (ga + gb) * LOG2E;
            g2e = (ge + gb) * LOG2E;
        }
        for (int c = 0; c < nc && ok; ++c) {
            const bool last = c + 1 == nc;
            if (!last) load_gates(c + 1, n_lam, n_ga, n_gb, n_ge);
            if (cq == 0) {
                s_g2[row] = g2;
                s_b[row] = ex2(g2e - g2);   // from this row's token to the end of its 16-block
            }
            if (ok) ok = mbar_wait_ab(&bars[OB_NX], c & 1, s_abort);
            fence_async_smem();
            tc_fence_before();
            ok = named_and(1, OUT_CHAIN, ok);
            tc_fence_after();
            if (!ok) break;
            const float gam = ex2(g2);

            // product 1: X1 = Q K^T, X2 = Q Kbar^T
            if (issuer()) {
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    mma_bf16(taddr + X1, kmajor_desc(uQ, 128, k), kmajor_desc(uK, 128, k), id_kk, k > 0);
                    mma_bf16(taddr + X2, kmajor_desc(uQ, 128, k), kmajor_desc(uN, 128, k), id_kk, k > 0);
                }
                // E1 rewrites T_S once this product completes: the previous chunk's output
                // store must have read it (the commit below is only issued after that)
                bulk_wait_read_all();
                mma_commit(&bars[OB_MMA]);
                mma_commit(&bars[OB_F1]);
                issued = true;
            }
            wait_mma();
            {   // P1 = s (Q K^T) o Gamma
                float x[32];
                tmem_ld16x2(tl + X1, x);
                mask_scores(x, g2, scale);
                store_q<__half>(T_S, row, c0, x);
            }
            publish();
            if (!ok) break;
            // product 2: X1 = P1 A
            if (issuer()) {
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16(taddr + X1, kmajor_desc(uS, 128, k), mnmajor_desc(uA, 128, k), id_kn, k > 0);
                mma_commit(&bars[OB_MMA]);
            }
            wait_mma();
            {   // z = U(lam) o',  o' = s gamma_r (Q Kbar^T) + P1 A
                float x[32], y[32];
                tmem_ld16x2_pair(tl + X2, x, tl + X1, y);
                const float f = scale * gam;
#pragma unroll
                for (int i = 0; i < 32; ++i) x[i] = fmaf(f, x[i], y[i]);
                rotate_q<1>(x, hf, u, lam, sl);
                store_q<__half>(T_S, row, c0, x);
            }
            publish();
            if (!ok) break;
            // product 3: X1 = z M^T
            if (issuer()) {
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16(taddr + X1, kmajor_desc(uS, 128, k), kmajor_desc(uM, 128, k), id_kk, k > 0);
                mma_commit(&bars[OB_MMA]);
            }
            wait_mma();
            {   // p = softmax over the m active slots of l = z M^T; the staging tile (z is
                // consumed) holds the row reductions over the four column quarters
                float* red = reinterpret_cast<float*>(T_S);
                float x[32];
                tmem_ld16x2(tl + X1, x);
                float mx = -INFINITY;
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    if (!slot_off(c0, i, sl)) mx = fmaxf(mx, x[i]);
                red[128 * cq + row] = mx;
                named_sync(1, OUT_CHAIN);
                mx = fmaxf(fmaxf(red[row], red[128 + row]), fmaxf(red[256 + row], red[384 + row]));
                float sum = 0.f;
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    x[i] = slot_off(c0, i, sl) ? 0.f : ex2((x[i] - mx) * LOG2E);
                    sum += x[i];
                }
                red[512 + 128 * cq + row] = sum;
                named_sync(1, OUT_CHAIN);
                const float inv = 1.f / ((red[512 + row] + red[640 + row]) + (red[768 + row] + red[896 + row]));
#pragma unroll
                for (int i = 0; i < 32; ++i) x[i] *= inv;
                named_sync(1, OUT_CHAIN);   // every quarter has read its sums before p overwrites them
                store_q<__half>(T_S, row, c0, x);
            }
            publish();
            if (!ok) break;
            // product 4: X2 = p M
            if (issuer()) {
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16(taddr + X2, kmajor_desc(uS, 128, k), mnmajor_desc(uM, 128, k), id_kn, k > 0);
                mma_commit(&bars[OB_MMA]);
            }
            wait_mma();
            {   // o'' = U(-lam) (p M)
                float x[32];
                tmem_ld16x2(tl + X2, x);
                rotate_q<-1>(x, hf, u, lam, sl);
                store_q<__half>(T_S, row, c0, x);
            }
            publish();
            if (!ok) break;
            // product 5: X1 = O'' A^T, X2 = O'' Vbar (needs the Vbar snapshot: state ready)
            if (issuer()) {
                ok = mbar_wait_ab(&bars[OB_SR], c & 1, s_abort);
                if (ok) {
                    tc_fence_after();
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                        mma_bf16(taddr + X1, kmajor_desc(uS, 128, k), kmajor_desc(uA, 128, k), id_kk, k > 0);
                        mma_bf16(taddr + X2, kmajor_desc(uS, 128, k), mnmajor_desc(uN, 128, k), id_kn, k > 0);
                    }
                    mma_commit(&bars[OB_MMA]);
                    mma_commit(&bars[OB_F5]);
                }
            }
            wait_mma();
            {   // P2 = (O'' A^T) o Gamma
                float x[32];
                tmem_ld16x2(tl + X1, x);
                mask_scores(x, g2, 1.f);
                store_q<__half>(T_S, row, c0, x);
            }
            publish();
            if (!ok) break;
            // product 6: X1 = P2 V
            if (issuer()) {
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16(taddr + X1, kmajor_desc(uS, 128, k), mnmajor_desc(uV, 128, k), id_kn, k > 0);
                mma_commit(&bars[OB_MMA]);
                mma_commit(&bars[OB_F6]);
            }
            wait_mma();
            {   // o = gamma_r (O'' Vbar) + P2 V, staged in T_S (P2 is consumed) for a TMA store
                float x[32], y[32];
                tmem_ld16x2_pair(tl + X2, x, tl + X1, y);
                float fin = 0.f;   // a non-finite output makes the sum non-finite
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    x[i] = fmaf(gam, x[i], y[i]);
                    fin += x[i];
                }
                // an fp16 operand that overflowed (the Vbar snapshot) reaches o as inf / NaN
                if (!isfinite(fin)) flag_error(CYFA_ERR_RANGE);
                store_q<__nv_bfloat16>(T_S, row, c0, x);
            }
            publish();
            if (tid == 0) {
                issued = false;   // every product of the chunk has been waited for
                if (ok) {
                    const int r0 = b * s.T + (c_begin + c) * CT;
                    tma_store_3d(&to, T_S, 0, h, r0);
                    tma_store_3d(&to, T_S + TILE / 2, 64, h, r0);
                    bulk_commit();
                }
            }
            if (!last) {
                lam = n_lam;
                g2 = (n_ga + n_gb) * LOG2E;
                g2e = (n_ge + n_gb) * LOG2E;
                // the next chunk's Q and K (loaded once the state update had read T_Q, T_K)
                // become fp16 operands
                if (ok) ok = mbar_wait_ab(&bars[OB_QK], (c + 1) & 1, s_abort);
                if (ok) {
                    bf16_to_f16_q(T_Q, row, c0);
                    bf16_to_f16_q(T_K, row, c0);
                }
            }
        }
        if (!ok) *s_abort = 1;
        if (tid == 0 && issued) {   // a product may still be running: let it finish
            mma_commit(&bars[OB_END]);
            mbar_wait(&bars[OB_END], 0);
        }
        if (tid == 0) bulk_wait_all();
    }
    tc_fence_before();
    __syncthreads();
    if (tid < 32) tmem_dealloc(taddr, 512);
}

// M = R Phi (App. A.1 Eq. app-real-fourier: Phi[r][0] = 1/sqrt(m), Phi[r][2j-1] =
// sqrt(2/m) cos(2 pi j r / m), Phi[r][2j] = sqrt(2/m) sin(2 pi j r / m)) straight into fp16 with
// its Fourier (column) index in the tensor-core order; the padding row and column are zero.
// Block (group of 8 rows i, h), 128 threads: thread p owns Fourier column p and accumulates its 8
// rows over r in fp32, in the same order as the CUDA-core path's readout matrix.
__global__ void __launch_bounds__(128) readout_f16_kernel(const float* R, __half* Mb, Slots sl) {
    const int h = blockIdx.y, i0 = 8 * blockIdx.x, p = threadIdx.x;
    const int m = sl.m;                  // R is [H, m, m]; rows and columns m..127 of M are zero
    __shared__ float s_r[8][MA];
    __shared__ float s_c[MA], s_s[MA];   // cos / sin of 2 pi x / m, x = 0 .. m - 1
    for (int e = p; e < 8 * m; e += 128) {
        const int ii = e / m, r = e - ii * m;
        s_r[ii][r] = (i0 + ii < m) ? R[((size_t)h * m + i0 + ii) * m + r] : 0.f;
    }
    if (p < m) {
        float sv, cv;
        sincospif((float)p * sl.two_over_m, &sv, &cv);
        s_c[p] = cv;
        s_s[p] = sv;
    }
    __syncthreads();
    float acc[8];
#pragma unroll
    for (int ii = 0; ii < 8; ++ii) acc[ii] = 0.f;
    if (p == 0) {
        for (int r = 0; r < m; ++r)
#pragma unroll
            for (int ii = 0; ii < 8; ++ii) acc[ii] = fmaf(s_r[ii][r], sl.inv_sqrt_m, acc[ii]);
    } else if (p < m) {
        const int j = (p + 1) >> 1;
        const float* tab = (p & 1) ? s_c : s_s;
        int idx = 0;   // (j r) mod m
        for (int r = 0; r < m; ++r) {
            const float phi = sl.sqrt2_over_m * tab[idx];
#pragma unroll
            for (int ii = 0; ii < 8; ++ii) acc[ii] = fmaf(s_r[ii][r], phi, acc[ii]);
            idx += j;
            if (idx >= m) idx -= m;
        }
    }
#pragma unroll
    for (int ii = 0; ii < 8; ++ii) {
        const int i = i0 + ii;
        Mb[((size_t)h * MS + i) * MS + tc_slot(p)] = __float2half_rn(i < m ? acc[ii] : 0.f);
    }
}

// Total log-decay of every segment (sum of its chunks' 128-token totals), as seg_state_tc
// computes it; one warp per (segment, b*h).
__global__ void seg_decay_kernel(TcFwdArgs a, int segc) {
    const Shape s = a.s;
    const int seg = blockIdx.x, bh = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nct = s.T / CT, c_begin = seg * segc, nc = min(segc, nct - c_begin);
    const int lane = threadIdx.x;
    float tot = 0.f;
    if (lane < nc) {
        const int t0 = (c_begin + lane) * CT;
        tot = cum128(s, a.g, b, h, t0, t0 + CT - 1);
    }
    // the same order as seg_state_tc: acc over chunks from last to first
    float acc = 0.f;
    for (int c = nc - 1; c >= 0; --c) acc += __shfl_sync(0xffffffffu, tot, c);
    if (lane == 0) a.segG[(size_t)bh * a.nseg + seg] = acc;
}

constexpr int SEGC_DEFAULT = TC_SEGC;

}  // namespace

int tc_fwd_segments(const Shape& s) {
    const int nct = s.T / CT;
    return (nct + SEGC_DEFAULT - 1) / SEGC_DEFAULT;
}

// m >= 63: the fp16 operands' error in the clock gradient grows as 1 / sqrt(m) (fewer slots hold
// larger, more cancelling terms): rel-L2 1.1e-3 at m = 127, 3.1e-3 at m = 63, 1.1e-2 at m = 5;
// smaller m run on the fp32 CUDA-core kernels.
bool tc_fwd_supported(const Shape& s) {
    return s.bf16 && s.D == 128 && s.sl.m >= 63 && s.T % CT == 0;
}

bool tc_qkv_maps(const Shape& s, const void* q, const void* k, const void* v, CUtensorMap* mq,
                 CUtensorMap* mk, CUtensorMap* mv, unsigned box_rows) {
    const unsigned long long dims[3] = {128ull, (unsigned long long)s.H,
                                        (unsigned long long)s.B * s.T};
    const unsigned long long strides[2] = {128ull * 2, (unsigned long long)s.H * 128 * 2};
    const unsigned box[3] = {64, 1, box_rows};
    return (!mq || make_tmap_bf16(mq, q, 3, dims, strides, box)) &&
           (!mk || make_tmap_bf16(mk, k, 3, dims, strides, box)) &&
           (!mv || make_tmap_bf16(mv, v, 3, dims, strides, box));
}

bool tc_rows_map(CUtensorMap* map, const void* base, unsigned long long rows, bool f16,
                 unsigned box_rows) {
    const unsigned long long dims[2] = {128ull, rows};
    const unsigned long long str[1] = {256ull};
    const unsigned box[2] = {64, box_rows};
    return make_tmap_bf16(map, base, 2, dims, str, box, f16);
}

cudaError_t launch_readout_f16(int H, const float* R, __half* Mb, const Slots& sl,
                               cudaStream_t st) {
    { LaunchScope ls_("readout_f16", st); readout_f16_kernel<<<dim3(MS / 8, H), 128, 0, st>>>(R, Mb, sl); }
    return cudaGetLastError();
}

cudaError_t launch_fwd_segment_states(const TcFwdArgs& a, const void* k, const void* v,
                                      cudaStream_t st) {
    const Shape& s = a.s;
    CUtensorMap mk, mv;
    if (!tc_qkv_maps(s, nullptr, k, v, nullptr, &mk, &mv)) return cudaErrorInvalidValue;
    const dim3 grid(s.B * s.H, a.nseg);   // heads fastest: CTAs that share token rows run together
    const int smA = 1024 + 12 * SEGC_DEFAULT * CT + 6 * TILE + 1024;
    auto kA = s.sl.m == 127 ? seg_state_tc<SEGC_DEFAULT, __half, Slots127>
                            : seg_state_tc<SEGC_DEFAULT, __half, Slots>;
    cudaFuncSetAttribute(kA, cudaFuncAttributeMaxDynamicSharedMemorySize, smA);
    { LaunchScope ls_("tc_seg_state", st); kA<<<grid, 512, smA, st>>>(mk, mv, a); }
    { LaunchScope ls_("tc_seg_scan", st); seg_scan_kernel<<<dim3(128, s.B * s.H), 256, 0, st>>>(a); }
    return cudaGetLastError();
}

cudaError_t launch_segment_decay(const TcFwdArgs& a, cudaStream_t st) {
    const Shape& s = a.s;
    { LaunchScope ls_("tc_seg_decay", st); seg_decay_kernel<<<dim3(a.nseg, s.B * s.H), 32, 0, st>>>(a, SEGC_DEFAULT); }
    return cudaGetLastError();
}

cudaError_t launch_fwd_tc(const TcFwdArgs& a, const void* q, const void* k, const void* v,
                          cudaStream_t st) {
    const Shape& s = a.s;
    const unsigned long long BH = (unsigned long long)s.B * s.H;
    CUtensorMap mq, mk, mv, mm, msnap, mo;
    if (!tc_qkv_maps(s, q, k, v, &mq, &mk, &mv) ||
        !tc_qkv_maps(s, a.o, nullptr, nullptr, &mo, nullptr, nullptr) ||
        !tc_rows_map(&mm, a.Mb, (unsigned long long)s.H * 128, true))
        return cudaErrorInvalidValue;
    // without a snapshot buffer the map is a valid placeholder over M that is never used
    if (!tc_rows_map(&msnap, a.snap ? (const void*)a.snap : (const void*)a.Mb,
                     a.snap ? BH * (s.T / CT) * 2 * 128 : (unsigned long long)s.H * 128, true))
        return cudaErrorInvalidValue;
    cudaError_t e = launch_fwd_segment_states(a, k, v, st);
    if (e != cudaSuccess) return e;
    const dim3 grid(s.B * s.H, a.nseg);   // heads fastest: CTAs that share token rows run together
    const int smC = 2048 + 7 * TILE + 1024;
    auto kC = s.sl.m == 127 ? seg_out_tc<SEGC_DEFAULT, Slots127> : seg_out_tc<SEGC_DEFAULT, Slots>;
    cudaFuncSetAttribute(kC, cudaFuncAttributeMaxDynamicSharedMemorySize, smC);
    { LaunchScope ls_("tc_seg_out", st); kC<<<grid, OUT_THREADS, smC, st>>>(mq, mk, mv, mm, msnap, mo, a); }
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
