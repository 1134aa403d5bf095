// fp32 SIMT chunk kernels of the CyFA operator (forward and backward).
//
// Chunk-wise two-pass form of App. B (Eqs. app-chunk-decay, app-chunk-rescale,
// app-temporal-writes, app-cyfa-key-chunk, app-cyfa-value-chunk) with the token-wise middle
// line of Sec. 3.3 Eq. cyfa-two-pass.  Every product accumulates in fp32 on the CUDA cores;
// this path serves fp32 inputs (and any input when exactness is wanted over speed).
//
// States are stored in the paper's orientation: Kbar [ms x dk] (= (S^K)^T of App. B) and
// Vbar [ms x dv], side by side as one [ms x 2D] row-major block per chunk (ms = 128 storage
// rows for m <= 127, 256 for larger m).
#include "simt_tiles.cuh"

namespace cyfa {

namespace {

// ---------------------------------------------------------------------------------------
// M = R Phi (padded to ms x ms with zero rows and columns m..ms-1) and its transpose.
// Phi is the real Fourier basis of App. A.1 Eq. app-real-fourier; R is [H, m, m].  Block (i, h)
// of ms threads: thread col forms M[i][col].
__global__ void __launch_bounds__(MS_MAX) readout_matrix_kernel(const float* R, float* M, float* MT,
                                                                Slots sl) {
    const int h = blockIdx.y, i = blockIdx.x, col = threadIdx.x;
    const int m = sl.m, ms = sl.ms;
    __shared__ float srow[MS_MAX], s_ct[MS_MAX], s_st[MS_MAX];
    srow[col] = (i < m && col < m) ? R[((size_t)h * m + i) * m + col] : 0.f;
    if (col < m) {   // cos / sin of 2 pi x / m for x = 0 .. m-1 (the entries of Phi)
        float sv, cv;
        sincospif((float)col * sl.two_over_m, &sv, &cv);
        s_ct[col] = cv;
        s_st[col] = sv;
    }
    __syncthreads();
    float acc = 0.f;
    if (i < m && col < m) {
        if (col == 0) {
            for (int r = 0; r < m; ++r) acc = fmaf(srow[r], sl.inv_sqrt_m, acc);
        } else {
            const int j = (col + 1) >> 1;
            const float* tab = (col & 1) ? s_ct : s_st;
            int idx = 0;   // (j r) mod m
            for (int r = 0; r < m; ++r) {
                acc = fmaf(srow[r], sl.sqrt2_over_m * tab[idx], acc);
                idx += j;
                if (idx >= m) idx -= m;
            }
        }
    }
    M[((size_t)h * ms + i) * ms + col] = acc;
    MT[((size_t)h * ms + col) * ms + i] = acc;
}

// ---------------------------------------------------------------------------------------
// Forward state pass: one block per (b, h, 64-column tile of [Kbar | Vbar], 128 of the MSZ
// storage rows); walks the chunks in order, writing the chunk-start state, then
// Kbar <- gamma^C Kbar + A->^T K (and V), App. B Eq. app-cyfa-key-chunk / app-cyfa-value-chunk
// (first lines).  The storage rows are independent in this recurrence.
template <int C, int MSZ, typename TI>
__global__ void __launch_bounds__(256) fwd_state_kernel(FwdArgs a) {
    constexpr int LDM = MSZ + 1, NCOL = 64, NJ = NCOL / 16;
    const Shape s = a.s;
    const int D = s.D, W = 2 * s.D;
    const int bh = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int col0 = blockIdx.x * NCOL;
    const int rz = 128 * blockIdx.z;   // first storage row of this block
    const bool isK = col0 < D;
    const TI* X = (const TI*)(isK ? a.k : a.v);
    const int xc0 = isK ? col0 : col0 - D;
    extern __shared__ float smem[];
    float* sA = smem;              // [C][LDM]
    float* sX = sA + C * LDM;      // [C][NCOL + 1]
    float* sg = sX + C * (NCOL + 1);
    float* slam = sg + C;
    float* sbeta = slam + C;
    if (!launch_ok(smem, sbeta + C)) return;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float S[8][NJ];
    const float* S0 = isK ? a.Kbar0 : a.Vbar0;
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < NJ; ++j)
            S[i][j] = S0 ? S0[((size_t)bh * MSZ + rz + ty + 16 * i) * D + xc0 + tx + 16 * j] : 0.f;
    const int nchunk = s.nchunk();
    for (int c = 0; c < nchunk; ++c) {
        float* dst = a.states + ((size_t)bh * nchunk + c) * MSZ * W;
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) dst[(rz + ty + 16 * i) * W + col0 + tx + 16 * j] = S[i][j];
        const int t0 = c * C;
        load_gates(s, a.lam, a.g, a.beta, b, h, t0, C, slam, sg, sbeta);
        stage_tok<C, NCOL>(sX, X, s, b, h, t0, xc0, 1.f);
        __syncthreads();
        const float gC = sg[C - 1];
        build_write_rows(sA, LDM, slam, sbeta, C, s.sl, [&](int r) { return expf(gC - sg[r]); });
        __syncthreads();
        const float decay = expf(gC);
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) S[i][j] *= decay;
        simt_mm<8, NJ>(S, C, [&](int row, int t) { return sA[t * LDM + rz + row]; },
                       [&](int t, int col) { return sX[t * (NCOL + 1) + col]; });
        __syncthreads();
    }
    float* F = isK ? a.Kout : a.Vout;
    if (F) {
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j)
                F[((size_t)bh * MSZ + rz + ty + 16 * i) * D + xc0 + tx + 16 * j] = S[i][j];
    }
}

// Forward outputs of one chunk (App. B, second lines of Eqs. app-cyfa-key-chunk and
// app-cyfa-value-chunk, with the middle readout between them).
template <int C, int D, int MSZ, typename TI>
__global__ void __launch_bounds__(256, (C == 64 && MSZ == 128) ? 2 : 1) fwd_out_kernel(FwdArgs a) {
    const Shape s = a.s;
    constexpr int LP = C + 1, TM = C / 16, LDM = MSZ + 1, NJ = MSZ / 16;
    const int c = blockIdx.x, bh = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nchunk = s.nchunk();
    const int t0 = c * C;
    extern __shared__ float smem[];
    float* sA = smem;            // [C][LDM]  write vectors; later staging
    float* sX = sA + C * LDM;    // [C][LDM]  staging, then O', then O''
    float* sP = sX + C * LDM;    // [C][LP]   masked intra-chunk scores
    float* sg = sP + C * LP;
    float* seg = sg + C;
    float* slam = seg + C;
    float* sbeta = slam + C;
    // staging of M^T / M for the middle readout: the score tile (free during the readout) when
    // it is large enough, else its own region
    float* sB = C * LP >= 32 * LDM ? sP : sbeta + C;
    if (!launch_ok(smem, sbeta + C + (C * LP >= 32 * LDM ? 0 : 32 * LDM))) return;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const float* Sst = a.states + ((size_t)bh * nchunk + c) * MSZ * (2 * D);
    const TI* Q = (const TI*)a.q;
    const TI* K = (const TI*)a.k;
    const TI* V = (const TI*)a.v;

    load_gates(s, a.lam, a.g, a.beta, b, h, t0, C, slam, sg, sbeta);
    __syncthreads();
    for (int r = threadIdx.x; r < C; r += blockDim.x) seg[r] = expf(sg[r]);
    build_write_rows(sA, LDM, slam, sbeta, C, s.sl, [](int) { return 1.f; });

    // P = (s Q K^T) o Gamma
    float acc[TM][TM];
    zero_acc(acc);
    for (int d0 = 0; d0 < D; d0 += 32) {
        __syncthreads();
        stage_tok<C>(sX, Q, s, b, h, t0, d0, 1.f);
        stage_tok<C>(sX + C * 33, K, s, b, h, t0, d0, 1.f);
        __syncthreads();
        simt_mm<TM, TM>(acc, 32, [&](int r, int kk) { return sX[r * 33 + kk]; },
                        [&](int kk, int t) { return sX[C * 33 + t * 33 + kk]; });
    }
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TM; ++j) {
            const int r = ty + 16 * i, t = tx + 16 * j;
            sP[r * LP + t] = (t <= r) ? acc[i][j] * s.scale * expf(sg[r] - sg[t]) : 0.f;
        }

    // O' = diag(gamma) (s Q) Kbar^T + P A  (the staged Q and Kbar columns fit in sX:
    // (C + MSZ) * 33 <= C * LDM for the (C, MSZ) instantiated)
    static_assert((C + MSZ) * 33 <= C * LDM, "Q / Kbar staging exceeds its tile");
    float o1[TM][NJ];
    zero_acc(o1);
    for (int d0 = 0; d0 < D; d0 += 32) {
        __syncthreads();
        stage_tok<C>(sX, Q, s, b, h, t0, d0, 1.f);
        stage_elems<MSZ * 32 / SIMT_THREADS>(
            MSZ * 32, [&](int e) { return Sst[(e >> 5) * (2 * D) + d0 + (e & 31)]; },
            [&](int e, float x) { sX[C * 33 + (e >> 5) * 33 + (e & 31)] = x; });
        __syncthreads();
        simt_mm<TM, NJ>(o1, 32, [&](int r, int kk) { return sX[r * 33 + kk]; },
                        [&](int kk, int i) { return sX[C * 33 + i * 33 + kk]; });
    }
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < NJ; ++j) o1[i][j] *= s.scale * seg[ty + 16 * i];
    simt_mm<TM, NJ>(o1, C, [&](int r, int t) { return sP[r * LP + t]; },
                    [&](int t, int i) { return sA[t * LDM + i]; });
    __syncthreads();
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < NJ; ++j) sX[(ty + 16 * i) * LDM + tx + 16 * j] = o1[i][j];
    __syncthreads();

    readout_rows_fwd<C, MSZ>(sX, sB, slam, a.M + (size_t)h * MSZ * MSZ,
                             a.MT + (size_t)h * MSZ * MSZ, s.sl);
    __syncthreads();

    // P = (O'' A^T) o Gamma
    zero_acc(acc);
    simt_mm<TM, TM>(acc, MSZ, [&](int r, int kk) { return sX[r * LDM + kk]; },
                    [&](int kk, int t) { return sA[t * LDM + kk]; });
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TM; ++j) {
            const int r = ty + 16 * i, t = tx + 16 * j;
            sP[r * LP + t] = (t <= r) ? acc[i][j] * expf(sg[r] - sg[t]) : 0.f;
        }

    // O = diag(gamma) O'' Vbar + P V
    constexpr int TN = D / 16;
    float o[TM][TN];
    zero_acc(o);
    float* sV = sA;  // staging [32][D+1]
    static_assert(32 * (D + 1) <= C * LDM, "V staging exceeds its tile");
    for (int i0 = 0; i0 < MSZ; i0 += 32) {
        __syncthreads();
        stage_elems<32 * D / SIMT_THREADS>(
            32 * D, [&](int e) { return Sst[(i0 + e / D) * (2 * D) + D + e % D]; },
            [&](int e, float x) { sV[(e / D) * (D + 1) + e % D] = x; });
        __syncthreads();
        simt_mm<TM, TN>(o, 32, [&](int r, int ii) { return sX[r * LDM + i0 + ii]; },
                        [&](int ii, int dd) { return sV[ii * (D + 1) + dd]; });
    }
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) o[i][j] *= seg[ty + 16 * i];
    for (int s0 = 0; s0 < C; s0 += 32) {
        __syncthreads();
        stage_elems<32 * D / SIMT_THREADS>(
            32 * D,
            [&](int e) { return ldf(V, (((size_t)b * s.T + t0 + s0 + e / D) * s.H + h) * D + e % D); },
            [&](int e, float x) { sV[(e / D) * (D + 1) + e % D] = x; });
        __syncthreads();
        simt_mm<TM, TN>(o, 32, [&](int r, int ss) { return sP[r * LP + s0 + ss]; },
                        [&](int ss, int dd) { return sV[ss * (D + 1) + dd]; });
    }
    TI* O = (TI*)a.o;
#pragma unroll
    for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            const int r = ty + 16 * i, dd = tx + 16 * j;
            stf(O, (((size_t)b * s.T + t0 + r) * s.H + h) * D + dd, o[i][j]);
        }
}

template <int C, int MSZ, typename TI>
cudaError_t launch_state(const FwdArgs& a, const char* name, cudaStream_t st) {
    const Shape& s = a.s;
    const size_t sm = (size_t)(C * (MSZ + 1) + C * 65 + 3 * C) * sizeof(float);
    auto k = fwd_state_kernel<C, MSZ, TI>;
    cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    { LaunchScope ls_(name, st); k<<<dim3(2 * s.D / 64, s.B * s.H, MSZ / 128), 256, sm, st>>>(a); }
    return cudaGetLastError();
}

template <int C, int D, int MSZ, typename TI>
cudaError_t fwd_dispatch(const FwdArgs& a, cudaStream_t st) {
    const Shape& s = a.s;
    cudaError_t e = launch_state<C, MSZ, TI>(a, "fwd_state", st);
    if (e != cudaSuccess) return e;
    constexpr int SB_EXTRA = C * (C + 1) >= 32 * (MSZ + 1) ? 0 : 32 * (MSZ + 1);
    const size_t sm_out = (size_t)(2 * C * (MSZ + 1) + C * (C + 1) + 4 * C + SB_EXTRA) * sizeof(float);
    auto kout = fwd_out_kernel<C, D, MSZ, TI>;
    cudaFuncSetAttribute(kout, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_out);
    { LaunchScope ls_("fwd_out", st); kout<<<dim3(s.nchunk(), s.B * s.H), 256, sm_out, st>>>(a); }
    return cudaGetLastError();
}

}  // namespace

cudaError_t simt_fwd_read_error(cudaStream_t st, int* err) { return read_simt_error(st, err); }

cudaError_t launch_readout_matrix(int H, const float* R, float* M, float* MT, const Slots& sl,
                                  cudaStream_t st) {
    { LaunchScope ls_("readout_matrix", st); readout_matrix_kernel<<<dim3(sl.ms, H), sl.ms, 0, st>>>(R, M, MT, sl); }
    return cudaGetLastError();
}

// State pass alone at the chunk length s.C: 64 or 128 with 128 storage rows (the forward's
// chunks and the backward's), 32 or 64 with 256.
cudaError_t launch_state_simt(const FwdArgs& a, cudaStream_t st) {
    const Shape& s = a.s;
#define CYFA_ST(CC, MM)                                                                    \
    if (s.C == CC && s.sl.ms == MM)                                                        \
        return s.bf16 ? launch_state<CC, MM, __nv_bfloat16>(a, "state_pass", st)          \
                      : launch_state<CC, MM, float>(a, "state_pass", st);
    CYFA_ST(64, 128)
    CYFA_ST(128, 128)
    CYFA_ST(32, 256)
    CYFA_ST(64, 256)
#undef CYFA_ST
    return cudaErrorInvalidValue;
}

// Chunk lengths walked: 64 or 128 with 128 storage rows (64 at d = 256), 64 with 256.
cudaError_t launch_fwd_simt(const FwdArgs& a, cudaStream_t st) {
    const Shape& s = a.s;
#define CYFA_FWD(CC, DD, MM)                                                             \
    if (s.C == CC && s.D == DD && s.sl.ms == MM)                                         \
        return s.bf16 ? fwd_dispatch<CC, DD, MM, __nv_bfloat16>(a, st)                   \
                      : fwd_dispatch<CC, DD, MM, float>(a, st);
    CYFA_FWD(64, 64, 128)
    CYFA_FWD(64, 128, 128)
    CYFA_FWD(128, 64, 128)
    CYFA_FWD(128, 128, 128)
    CYFA_FWD(64, 256, 128)
    CYFA_FWD(64, 64, 256)
    CYFA_FWD(64, 128, 256)
    CYFA_FWD(64, 256, 256)
#undef CYFA_FWD
    return cudaErrorInvalidValue;
}

}  // namespace cyfa
