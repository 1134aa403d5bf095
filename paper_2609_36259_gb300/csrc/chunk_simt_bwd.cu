// fp32 SIMT backward of the CyFA operator (chunk length 64 with 128 storage rows, 32 with 256).
//
// The forward (App. B Eqs. app-cyfa-key-chunk / app-cyfa-value-chunk with the middle line of
// Sec. 3.3 Eq. cyfa-two-pass) is differentiated chunk by chunk:
//   1. chunk-start states are recomputed (forward state pass);
//   2. bwd_intra1: per chunk, recompute O' and O''; dO'' = gamma o (dO Vbar^T) + (dO V^T o Gamma) A;
//      the middle readout's gradient gives dO'; dQ = s [gamma o (dO' Kbar) + (dO' A^T o Gamma) K];
//   3. a reverse chunk scan of the state adjoints, D_c = gamma^C D_{c+1} + sum_r gamma^r [dO'_r q~_r^T | o''_r dO_r^T];
//   4. bwd_intra2: per chunk, dK, dV and dA (the write-vector gradient of both passes) from the
//      intra-chunk scores and the adjoint D_{c+1} of the chunk-end state;
//   5. reverse cumulative sums over tokens: d log alpha_s = sum_{t>=s} dG_t and
//      d delta_s = sum_{t>=s} d lambda_t (App. D.1 Eq. app-clock-gradient-accumulation), then the
//      activation derivatives to the logits.
// Per token, with the scalar-gated identity dG_t = <q_t, dq_t> - <k_t, dk_t> applied to each pass
// (key pass: q = s q, k = k, v = a; value pass: q = o'', k = a, v = v), and, from the three places
// lambda_t enters (a_t = beta U(-lambda) b, z_t = U(lambda) o', o'' = U(-lambda) y):
//   d lambda_t = -<da_t, Omega a_t> + <dz_t, Omega z_t> - <do''_t, Omega o''_t>,
// Omega the generator of U (blocks (2 pi j / m) [[0, -1], [1, 0]]).
#include "simt_tiles.cuh"

namespace cyfa {

namespace {

// Tile geometry for MSZ storage rows: chunks of CB tokens (64 with 128 rows; 32 with 256, so
// that five [CB][MSZ + 1] tiles still fit in shared memory); TMB rows per thread.
template <int MSZ>
struct Geo {
    static constexpr int CB = MSZ == 128 ? BWD_C : BWD_C256;
    static constexpr int LPB = CB + 1, TMB = CB / 16, LDM = MSZ + 1, NJ = MSZ / 16;
    static constexpr int NP = MSZ / 64, NE = MSZ / 32;
};
// Floats of the staging tile: the larger of a [CB][MSZ + 1] tile, the Q / Kbar column staging
// ((CB + MSZ) x 33) and the state-row staging (32 x (D + 1)).
template <int D, int MSZ>
__host__ __device__ constexpr int staging_floats() {
    constexpr int a = Geo<MSZ>::CB * Geo<MSZ>::LDM, b = (Geo<MSZ>::CB + MSZ) * 33, c = 32 * (D + 1);
    return a > b ? (a > c ? a : c) : (b > c ? b : c);
}

// 2 pi j / m, the rotation rate of pair j
__device__ __forceinline__ float freq(int j, const Slots& sl) {
    return (6.283185307179586f * sl.inv_m) * (float)j;
}

// <x, Omega y> for MSZ-vectors in shared memory, summed over the warp (pairs j = lane+1+32u).
template <int MSZ>
__device__ __forceinline__ float warp_omega_dot(const float* x, const float* y, int lane,
                                                const Slots& sl) {
    float acc = 0.f;
#pragma unroll
    for (int u = 0; u < Geo<MSZ>::NP; ++u) {
        const int j = lane + 1 + 32 * u;
        if (j <= sl.npair)
            acc += freq(j, sl) * (x[2 * j] * y[2 * j - 1] - x[2 * j - 1] * y[2 * j]);
    }
    return warp_sum(acc);
}

// The middle readout and its gradient for the CB rows of a chunk, as products of the row blocks
// with M^T and M (global [MSZ][MSZ], zero beyond the m active rows and columns):
//   z = U(lam) o',  dy = U(lam) do''             rows of sZ and sG, in place
//   l = M z,  dp = M dy                          one pass over M^T
//   p = softmax(l) over the m active slots,  dl = p o (dp - <p, dp>)
//   y = M^T p,  dz = M^T dl                      one pass over M (p staged in sY, dl in sW)
//   o'' = U(-lam) y into sY,  do' = U(-lam) dz into sG
// with the row scalars sdG[r] = <o'', do''> = <y, dy> and
// sdL[r] = <dz, Omega z> - <do'', Omega o''> = <dz, Omega z> - <dy, Omega y> (U is orthogonal
// and commutes with Omega).  Entries beyond the m active ones are zero in every row.  With gz
// non-null the rows of z, p, dy, dl (for dR) go to gz / gp / gdy / gdl + MSZ r.  sW is a
// [CB][MSZ + 1] scratch tile and sB the [32][MSZ + 1] staging of M^T and M.  One block
// barrier at entry (the caller's rows are complete); the results are complete after the
// caller's next barrier.
template <int MSZ>
__device__ __noinline__ void readout_rows_bwd(float* sZ, float* sY, float* sG, float* sW, float* sB,
                                              const float* slam, const float* M, const float* MT,
                                              float* sdG, float* sdL, float* gz, float* gp,
                                              float* gdy, float* gdl, const Slots& sl) {
    using G = Geo<MSZ>;
    constexpr int CB = G::CB, LDM = G::LDM, NP = G::NP, NE = G::NE, TMB = G::TMB, NJ = G::NJ;
    constexpr int NW = SIMT_THREADS / 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int npair = sl.npair, m = sl.m;
    const int K = (m + 31) & ~31;   // the products run over the active entries in steps of 32
    __syncthreads();
    for (int r = warp; r < CB; r += NW) {   // z, dy; inactive entries zeroed (read up to K)
        float* z = sZ + r * LDM;
        float* y = sG + r * LDM;
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
                const float gc = y[2 * j - 1], gs = y[2 * j];
                y[2 * j - 1] = cs * gc - sn * gs;
                y[2 * j] = sn * gc + cs * gs;
            } else if (j < MSZ / 2) {
                z[2 * j - 1] = z[2 * j] = 0.f;
                y[2 * j - 1] = y[2 * j] = 0.f;
            }
        }
        if (lane == 0) z[MSZ - 1] = y[MSZ - 1] = 0.f;
    }
    // logits and their adjoint (the row ty + 16 i lives on the 16 threads of a half warp)
    float ldp[2][TMB][NJ];
    zero_acc(ldp[0]);
    zero_acc(ldp[1]);
    rows_times_gmat<2, TMB, MSZ>(ldp, sB, sZ, sG, MT, K);
    float(&l)[TMB][NJ] = ldp[0];
    float(&dp)[TMB][NJ] = ldp[1];
#pragma unroll
    for (int i = 0; i < TMB; ++i) {
        float mx = -INFINITY;
#pragma unroll
        for (int j = 0; j < NJ; ++j)
            if (tx + 16 * j < m) mx = fmaxf(mx, l[i][j]);
        mx = half_warp_max(mx);
        float sum = 0.f;
#pragma unroll
        for (int j = 0; j < NJ; ++j) {
            l[i][j] = tx + 16 * j < m ? expf(l[i][j] - mx) : 0.f;
            sum += l[i][j];
        }
        const float inv = 1.f / half_warp_sum(sum);
        float pdp = 0.f;
#pragma unroll
        for (int j = 0; j < NJ; ++j) {
            l[i][j] *= inv;
            pdp = fmaf(l[i][j], dp[i][j], pdp);
        }
        pdp = half_warp_sum(pdp);
#pragma unroll
        for (int j = 0; j < NJ; ++j) dp[i][j] = l[i][j] * (dp[i][j] - pdp);
    }
#pragma unroll
    for (int i = 0; i < TMB; ++i)
#pragma unroll
        for (int j = 0; j < NJ; ++j) {
            const int r = ty + 16 * i, c = tx + 16 * j;
            sY[r * LDM + c] = l[i][j];
            sW[r * LDM + c] = dp[i][j];
            if (gz) {
                gp[(size_t)r * MSZ + c] = l[i][j];
                gdl[(size_t)r * MSZ + c] = dp[i][j];
            }
        }
    float ydz[2][TMB][NJ];
    zero_acc(ydz[0]);
    zero_acc(ydz[1]);
    rows_times_gmat<2, TMB, MSZ>(ydz, sB, sY, sW, M, K);
    const float(&y)[TMB][NJ] = ydz[0];
    const float(&dz)[TMB][NJ] = ydz[1];
    __syncthreads();   // p and dl have been read
#pragma unroll
    for (int i = 0; i < TMB; ++i)
#pragma unroll
        for (int j = 0; j < NJ; ++j) {
            const int r = ty + 16 * i, c = tx + 16 * j;
            sY[r * LDM + c] = y[i][j];
            sW[r * LDM + c] = dz[i][j];
        }
    __syncthreads();
    for (int r = warp; r < CB; r += NW) {
        const float* z = sZ + r * LDM;
        const float* w = sW + r * LDM;   // dz
        float* yv = sY + r * LDM;        // y, then o''
        float* g = sG + r * LDM;         // dy, then do'
        float g1 = 0.f;
#pragma unroll
        for (int v = 0; v < NE; ++v) {
            const int e = lane + 32 * v;
            g1 = fmaf(yv[e], g[e], g1);
            if (gz) {
                gz[(size_t)r * MSZ + e] = z[e];
                gdy[(size_t)r * MSZ + e] = g[e];
            }
        }
        g1 = warp_sum(g1);
        __syncwarp();   // the row's entries have been read before their pairs are rewritten
        const float lam = slam[r];
        float om = 0.f;
#pragma unroll
        for (int u = 0; u < NP; ++u) {
            const int j = lane + 1 + 32 * u;
            if (j <= npair) {
                float sn, cs;
                sincospif(phase_pi_m(lam, j, sl), &sn, &cs);
                const float yc = yv[2 * j - 1], ys = yv[2 * j];
                const float gc = g[2 * j - 1], gs = g[2 * j];
                const float dc = w[2 * j - 1], ds = w[2 * j];
                const float zc = z[2 * j - 1], zs = z[2 * j];
                om += freq(j, sl) * ((ds * zc - dc * zs) - (gs * yc - gc * ys));
                yv[2 * j - 1] = cs * yc + sn * ys;
                yv[2 * j] = -sn * yc + cs * ys;
                g[2 * j - 1] = cs * dc + sn * ds;
                g[2 * j] = -sn * dc + cs * ds;
            } else if (j < MSZ / 2) {
                g[2 * j - 1] = g[2 * j] = 0.f;
            }
        }
        om = warp_sum(om);
        if (lane == 0) {
            g[0] = w[0];
            g[MSZ - 1] = 0.f;
            sdG[r] = g1;
            sdL[r] = om;
        }
    }
}

// sP[r][t] = mul * (sum_k X(r,k) Y(t,k)) * exp(g_r - g_t) for t <= r, else 0  (r, t < CB)
template <int MSZ, class FX, class FY>
__device__ __forceinline__ void masked_scores(float* sP, const float* sg, int K, float mul,
                                              const FX& fx, const FY& fy) {
    using G = Geo<MSZ>;
    constexpr int TMB = G::TMB;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[TMB][TMB];
    zero_acc(acc);
    simt_mm<TMB, TMB>(acc, K, fx, fy);
#pragma unroll
    for (int i = 0; i < TMB; ++i)
#pragma unroll
        for (int j = 0; j < TMB; ++j) {
            const int r = ty + 16 * i, t = tx + 16 * j;
            sP[r * G::LPB + t] = (t <= r) ? acc[i][j] * mul * expf(sg[r] - sg[t]) : 0.f;
        }
}

// masked scores from two token tensors staged 32 columns at a time through sS
template <int MSZ, typename TI>
__device__ __forceinline__ void masked_scores_tok(float* sP, float* sS, const float* sg,
                                                  const TI* X, const TI* Y, const Shape& s, int b,
                                                  int h, int t0, float mul) {
    using G = Geo<MSZ>;
    constexpr int TMB = G::TMB, CB = G::CB;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[TMB][TMB];
    zero_acc(acc);
    for (int d0 = 0; d0 < s.D; d0 += 32) {
        __syncthreads();
        stage_tok<CB>(sS, X, s, b, h, t0, d0, 1.f);
        stage_tok<CB>(sS + CB * 33, Y, s, b, h, t0, d0, 1.f);
        __syncthreads();
        simt_mm<TMB, TMB>(acc, 32, [&](int r, int kk) { return sS[r * 33 + kk]; },
                          [&](int kk, int t) { return sS[CB * 33 + t * 33 + kk]; });
    }
#pragma unroll
    for (int i = 0; i < TMB; ++i)
#pragma unroll
        for (int j = 0; j < TMB; ++j) {
            const int r = ty + 16 * i, t = tx + 16 * j;
            sP[r * G::LPB + t] = (t <= r) ? acc[i][j] * mul * expf(sg[r] - sg[t]) : 0.f;
        }
}

// acc[r][i] += sum_d X[r][d] * Sst[i][coff + d]  (X a token tensor, Sst a [MSZ][2D] state block)
template <int MSZ, typename TI>
__device__ __forceinline__ void tok_times_stateT(float (&acc)[Geo<MSZ>::TMB][Geo<MSZ>::NJ],
                                                 float* sS, const TI* X, const float* Sst,
                                                 int coff, const Shape& s, int b, int h, int t0) {
    using G = Geo<MSZ>;
    constexpr int CB = G::CB;
    for (int d0 = 0; d0 < s.D; d0 += 32) {
        __syncthreads();
        stage_tok<CB>(sS, X, s, b, h, t0, d0, 1.f);
        stage_elems<MSZ * 32 / SIMT_THREADS>(
            MSZ * 32, [&](int e) { return Sst[(e >> 5) * (2 * s.D) + coff + d0 + (e & 31)]; },
            [&](int e, float x) { sS[CB * 33 + (e >> 5) * 33 + (e & 31)] = x; });
        __syncthreads();
        simt_mm<G::TMB, G::NJ>(acc, 32, [&](int r, int kk) { return sS[r * 33 + kk]; },
                               [&](int kk, int i) { return sS[CB * 33 + i * 33 + kk]; });
    }
}

// acc[r][dd] += sum_i Y(r, i) * Sst[i][coff + dd]  (Y rows in shared memory with stride MSZ + 1)
template <int MSZ, int TN>
__device__ __forceinline__ void rows_times_state(float (&acc)[Geo<MSZ>::TMB][TN], float* sS,
                                                 const float* Y, const float* Sst, int coff) {
    using G = Geo<MSZ>;
    constexpr int D = 16 * TN;   // the head dimension
    for (int i0 = 0; i0 < MSZ; i0 += 32) {
        __syncthreads();
        stage_elems<32 * D / SIMT_THREADS>(
            32 * D, [&](int e) { return Sst[(i0 + e / D) * (2 * D) + coff + e % D]; },
            [&](int e, float x) { sS[(e / D) * (D + 1) + e % D] = x; });
        __syncthreads();
        simt_mm<G::TMB, TN>(acc, 32, [&](int r, int ii) { return Y[r * G::LDM + i0 + ii]; },
                            [&](int ii, int dd) { return sS[ii * (D + 1) + dd]; });
    }
}

// acc[r][dd] += sum_t P(r, t) * X[t][dd]  with P given by an accessor (K = CB tokens)
template <int MSZ, int TN, typename TI, class FP>
__device__ __forceinline__ void scores_times_tok(float (&acc)[Geo<MSZ>::TMB][TN], float* sS,
                                                 const FP& fp, const TI* X, const Shape& s,
                                                 int b, int h, int t0, float mul) {
    using G = Geo<MSZ>;
    constexpr int D = 16 * TN;   // the head dimension (s.D)
    for (int s0 = 0; s0 < G::CB; s0 += 32) {
        __syncthreads();
        stage_elems<32 * D / SIMT_THREADS>(
            32 * D,
            [&](int e) {
                return mul * ldf(X, (((size_t)b * s.T + t0 + s0 + e / D) * s.H + h) * D + e % D);
            },
            [&](int e, float x) { sS[(e / D) * (D + 1) + e % D] = x; });
        __syncthreads();
        simt_mm<G::TMB, TN>(acc, 32, [&](int r, int ss) { return fp(r, s0 + ss); },
                            [&](int ss, int dd) { return sS[ss * (D + 1) + dd]; });
    }
}

// ---------------------------------------------------------------------------------------
template <int D, int MSZ, typename TI>
__global__ void __launch_bounds__(256) bwd_intra1_kernel(BwdArgs a) {
    using G = Geo<MSZ>;
    constexpr int CB = G::CB, LDM = G::LDM, LPB = G::LPB, TMB = G::TMB, NJ = G::NJ;
    const Shape s = a.s;
    constexpr int TN = D / 16;
    const int c = blockIdx.x, bh = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nchunk = s.nchunk(), t0 = c * CB;
    extern __shared__ float smem[];
    float* sA = smem;
    float* sO1 = sA + CB * LDM;
    float* sO2 = sO1 + CB * LDM;
    float* sD = sO2 + CB * LDM;
    float* sS = sD + CB * LDM;                      // staging
    float* sP = sS + staging_floats<D, MSZ>();
    float* sg = sP + CB * LPB;
    float* seg = sg + CB;
    float* slam = seg + CB;
    float* sbeta = slam + CB;
    float* sdG = sbeta + CB;
    float* sdL = sdG + CB;
    float* sB = sdL + CB;                           // [32][MSZ + 1] staging of M^T / M
    if (!launch_ok(smem, sB + 32 * LDM)) return;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const float* Sst = a.states + ((size_t)bh * nchunk + c) * MSZ * (2 * D);
    const float* Mh = a.M + (size_t)h * MSZ * MSZ;
    const float* MTh = a.MT + (size_t)h * MSZ * MSZ;
    const TI* Q = (const TI*)a.q;
    const TI* K = (const TI*)a.k;
    const TI* V = (const TI*)a.v;
    const TI* dO = (const TI*)a.dO;

    load_gates(s, a.lam, a.g, a.beta, b, h, t0, CB, slam, sg, sbeta);
    __syncthreads();
    for (int r = threadIdx.x; r < CB; r += blockDim.x) seg[r] = expf(sg[r]);
    build_write_rows(sA, LDM, slam, sbeta, CB, s.sl, [](int) { return 1.f; });

    // O' = s gamma o (Q Kbar^T) + (s Q K^T o Gamma) A
    masked_scores_tok<MSZ>(sP, sS, sg, Q, K, s, b, h, t0, s.scale);
    {
        float o1[TMB][NJ];
        zero_acc(o1);
        tok_times_stateT<MSZ>(o1, sS, Q, Sst, 0, s, b, h, t0);
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) o1[i][j] *= s.scale * seg[ty + 16 * i];
        simt_mm<TMB, NJ>(o1, CB, [&](int r, int t) { return sP[r * LPB + t]; },
                         [&](int t, int i) { return sA[t * LDM + i]; });
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) sO1[(ty + 16 * i) * LDM + tx + 16 * j] = o1[i][j];
    }
    __syncthreads();

    // dO'' = gamma o (dO Vbar^T) + (dO V^T o Gamma) A
    masked_scores_tok<MSZ>(sP, sS, sg, dO, V, s, b, h, t0, 1.f);
    {
        float g2[TMB][NJ];
        zero_acc(g2);
        tok_times_stateT<MSZ>(g2, sS, dO, Sst, D, s, b, h, t0);
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) g2[i][j] *= seg[ty + 16 * i];
        simt_mm<TMB, NJ>(g2, CB, [&](int r, int t) { return sP[r * LPB + t]; },
                         [&](int t, int i) { return sA[t * LDM + i]; });
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) sD[(ty + 16 * i) * LDM + tx + 16 * j] = g2[i][j];
    }
    {   // the middle readout (o'' into sO2) and its gradient (do' into sD); sO1 ends as z
        const size_t rowbase = ((size_t)bh * s.T + t0) * MSZ;
        const bool dr = a.mZ != nullptr;
        readout_rows_bwd<MSZ>(sO1, sO2, sD, sS, sB, slam, Mh, MTh, sdG, sdL,
                              dr ? a.mZ + rowbase : nullptr, dr ? a.mP + rowbase : nullptr,
                              dr ? a.mDY + rowbase : nullptr, dr ? a.mDL + rowbase : nullptr, s.sl);
    }
    __syncthreads();

    // dQ~ = gamma o (dO' Kbar) + (dO' A^T o Gamma) K ;  dq = s dQ~
    masked_scores<MSZ>(sP, sg, MSZ, 1.f, [&](int r, int kk) { return sD[r * LDM + kk]; },
                       [&](int kk, int t) { return sA[t * LDM + kk]; });
    {
        float dqa[TMB][TN];
        zero_acc(dqa);
        rows_times_state<MSZ, TN>(dqa, sS, sD, Sst, 0);
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) dqa[i][j] *= seg[ty + 16 * i];
        scores_times_tok<MSZ, TN>(dqa, sS, [&](int r, int t) { return sP[r * LPB + t]; }, K, s,
                                  b, h, t0, 1.f);
        TI* dQ = (TI*)a.dq;
#pragma unroll
        for (int i = 0; i < TMB; ++i) {
            const int r = ty + 16 * i;
            const size_t row = (((size_t)b * s.T + t0 + r) * s.H + h) * D + tx;
            float qv[TN];   // the row's q, loaded before any store of dq
#pragma unroll
            for (int j = 0; j < TN; ++j) qv[j] = ldf(Q, row + 16 * j);
            float part = 0.f;
#pragma unroll
            for (int j = 0; j < TN; ++j) {
                part += qv[j] * dqa[i][j];             // <q, dq~ / s> * s = <q~, dq~>
                stf(dQ, row + 16 * j, s.scale * dqa[i][j]);
            }
            part = half_warp_sum(part) * s.scale;
            if (tx == 0) sdG[r] += part;
        }
    }
    __syncthreads();
    // stash o'' and dL/do' for the adjoint scan and the second intra-chunk pass
    float* o2 = a.o2 + ((size_t)bh * s.T + t0) * MSZ;
    float* do1 = a.do1 + ((size_t)bh * s.T + t0) * MSZ;
    for (int e = threadIdx.x; e < CB * MSZ; e += blockDim.x) {
        const int r = e / MSZ, i = e % MSZ;
        o2[e] = sO2[r * LDM + i];
        do1[e] = sD[r * LDM + i];
    }
    const size_t BTH = (size_t)s.B * s.T * s.H;
    for (int r = threadIdx.x; r < CB; r += blockDim.x) {
        const size_t gi = ((size_t)b * s.T + t0 + r) * s.H + h;
        a.tok[gi] = sdG[r];
        a.tok[BTH + gi] = sdL[r];
    }
}

// Reverse scan of the state adjoints, one block per (b, h, 64-column tile of [D^K | D^V], 128
// of the MSZ storage rows).  Stores, for every chunk c, the adjoint of the state at the end of
// chunk c.
template <int MSZ, typename TI>
__global__ void __launch_bounds__(256) adj_state_kernel(BwdArgs a) {
    using G = Geo<MSZ>;
    constexpr int CB = G::CB, LDM = G::LDM, NCOL = 64, NJ = NCOL / 16;
    const Shape s = a.s;
    const int D = s.D, W = 2 * s.D;
    const int bh = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int col0 = blockIdx.x * NCOL;
    const int rz = 128 * blockIdx.z;   // first storage row of this block
    const bool isK = col0 < D;
    const int xc0 = isK ? col0 : col0 - D;
    const TI* X = (const TI*)(isK ? a.q : a.dO);
    const float* Y = isK ? a.do1 : a.o2;
    const float xmul = isK ? s.scale : 1.f;
    extern __shared__ float smem[];
    float* sY = smem;            // [CB][LDM]
    float* sX = sY + CB * LDM;   // [CB][NCOL + 1]
    float* sg = sX + CB * (NCOL + 1);
    if (!launch_ok(smem, sg + CB)) return;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float S[8][NJ];
    zero_acc(S);
    const int nchunk = s.nchunk();
    for (int c = nchunk - 1; c >= 0; --c) {
        float* dst = a.adj + ((size_t)bh * nchunk + c) * MSZ * W;
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) dst[(rz + ty + 16 * i) * W + col0 + tx + 16 * j] = S[i][j];
        const int t0 = c * CB;
        __syncthreads();
        const float gb = g_base(s, a.g, b, h, t0, CB);
        for (int r = threadIdx.x; r < CB; r += blockDim.x)
            sg[r] = a.g[((size_t)b * s.T + t0 + r) * s.H + h] - gb;
        stage_tok<CB, NCOL>(sX, X, s, b, h, t0, xc0, xmul);
        __syncthreads();
        const float* Yc = Y + ((size_t)bh * s.T + t0) * MSZ;
        stage_elems<CB * MSZ / SIMT_THREADS>(
            CB * MSZ, [&](int e) { return Yc[e] * expf(sg[e / MSZ]); },
            [&](int e, float x) { sY[(e / MSZ) * LDM + e % MSZ] = x; });
        __syncthreads();
        const float decay = expf(sg[CB - 1]);
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) S[i][j] *= decay;
        simt_mm<8, NJ>(S, CB, [&](int row, int t) { return sY[t * LDM + rz + row]; },
                       [&](int t, int col) { return sX[t * (NCOL + 1) + col]; });
    }
}

template <int D, int MSZ, typename TI>
__global__ void __launch_bounds__(256) bwd_intra2_kernel(BwdArgs a) {
    using G = Geo<MSZ>;
    constexpr int CB = G::CB, LDM = G::LDM, LPB = G::LPB, TMB = G::TMB, NJ = G::NJ;
    const Shape s = a.s;
    constexpr int TN = D / 16;
    const int c = blockIdx.x, bh = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int nchunk = s.nchunk(), t0 = c * CB;
    extern __shared__ float smem[];
    float* sA = smem;
    float* sY1 = sA + CB * LDM;    // dL/do'
    float* sY2 = sY1 + CB * LDM;   // o''
    float* sDA = sY2 + CB * LDM;   // dL/da
    float* sS = sDA + CB * LDM;    // staging
    float* sP = sS + staging_floats<D, MSZ>();
    float* sg = sP + CB * LPB;
    float* sfw = sg + CB;
    float* slam = sfw + CB;
    float* sbeta = slam + CB;
    float* sdG = sbeta + CB;
    if (!launch_ok(smem, sdG + CB)) return;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const float* Dst = a.adj + ((size_t)bh * nchunk + c) * MSZ * (2 * D);
    const TI* Q = (const TI*)a.q;
    const TI* K = (const TI*)a.k;
    const TI* V = (const TI*)a.v;
    const TI* dO = (const TI*)a.dO;
    const size_t tokbase = ((size_t)b * s.T + t0) * s.H + h;

    load_gates(s, a.lam, a.g, a.beta, b, h, t0, CB, slam, sg, sbeta);
    {
        const float* y1 = a.do1 + ((size_t)bh * s.T + t0) * MSZ;
        const float* y2 = a.o2 + ((size_t)bh * s.T + t0) * MSZ;
        stage_elems<CB * MSZ / SIMT_THREADS>(
            CB * MSZ, [&](int e) { return y1[e]; },
            [&](int e, float x) { sY1[(e / MSZ) * LDM + e % MSZ] = x; });
        stage_elems<CB * MSZ / SIMT_THREADS>(
            CB * MSZ, [&](int e) { return y2[e]; },
            [&](int e, float x) { sY2[(e / MSZ) * LDM + e % MSZ] = x; });
    }
    __syncthreads();
    for (int r = threadIdx.x; r < CB; r += blockDim.x) {
        sfw[r] = expf(sg[CB - 1] - sg[r]);
        sdG[r] = 0.f;
    }
    build_write_rows(sA, LDM, slam, sbeta, CB, s.sl, [](int) { return 1.f; });
    __syncthreads();

    // dK = P3^T (s Q) + diag(fw) A D^K,  P3 = (dO' A^T) o Gamma
    masked_scores<MSZ>(sP, sg, MSZ, 1.f, [&](int r, int kk) { return sY1[r * LDM + kk]; },
                       [&](int kk, int t) { return sA[t * LDM + kk]; });
    {
        float acc[TMB][TN];
        zero_acc(acc);
        rows_times_state<MSZ, TN>(acc, sS, sA, Dst, 0);
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) acc[i][j] *= sfw[ty + 16 * i];
        scores_times_tok<MSZ, TN>(acc, sS, [&](int t, int r) { return sP[r * LPB + t]; }, Q, s,
                                  b, h, t0, s.scale);
        TI* dK = (TI*)a.dk;
#pragma unroll
        for (int i = 0; i < TMB; ++i) {
            const int t = ty + 16 * i;
            const size_t row = (tokbase + (size_t)t * s.H) * D + tx;
            float kv[TN];   // the row's k, loaded before any store of dk
#pragma unroll
            for (int j = 0; j < TN; ++j) kv[j] = ldf(K, row + 16 * j);
            float part = 0.f;
#pragma unroll
            for (int j = 0; j < TN; ++j) {
                part += kv[j] * acc[i][j];
                stf(dK, row + 16 * j, acc[i][j]);
            }
            part = half_warp_sum(part);
            if (tx == 0) sdG[t] -= part;
        }
    }
    // dV = P2^T dO + diag(fw) A D^V,  P2 = (O'' A^T) o Gamma
    __syncthreads();
    masked_scores<MSZ>(sP, sg, MSZ, 1.f, [&](int r, int kk) { return sY2[r * LDM + kk]; },
                       [&](int kk, int t) { return sA[t * LDM + kk]; });
    {
        float acc[TMB][TN];
        zero_acc(acc);
        rows_times_state<MSZ, TN>(acc, sS, sA, Dst, D);
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) acc[i][j] *= sfw[ty + 16 * i];
        scores_times_tok<MSZ, TN>(acc, sS, [&](int t, int r) { return sP[r * LPB + t]; }, dO, s,
                                  b, h, t0, 1.f);
        TI* dV = (TI*)a.dv;
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j)
                stf(dV, (tokbase + (size_t)(ty + 16 * i) * s.H) * D + tx + 16 * j, acc[i][j]);
    }
    // dA^V = P4^T O'' + diag(fw) V (D^V)^T,  P4 = (dO V^T) o Gamma
    masked_scores_tok<MSZ>(sP, sS, sg, dO, V, s, b, h, t0, 1.f);
    {
        float acc[TMB][NJ];
        zero_acc(acc);
        tok_times_stateT<MSZ>(acc, sS, V, Dst, D, s, b, h, t0);
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) acc[i][j] *= sfw[ty + 16 * i];
        simt_mm<TMB, NJ>(acc, CB, [&](int t, int r) { return sP[r * LPB + t]; },
                         [&](int r, int i) { return sY2[r * LDM + i]; });
#pragma unroll
        for (int i = 0; i < TMB; ++i) {
            const int t = ty + 16 * i;
            float part = 0.f;
#pragma unroll
            for (int j = 0; j < NJ; ++j) {
                sDA[t * LDM + tx + 16 * j] = acc[i][j];
                part += sA[t * LDM + tx + 16 * j] * acc[i][j];
            }
            part = half_warp_sum(part);
            if (tx == 0) sdG[t] -= part;
        }
    }
    // dA^K = P1^T dO' + diag(fw) K (D^K)^T,  P1 = (s Q K^T) o Gamma
    masked_scores_tok<MSZ>(sP, sS, sg, Q, K, s, b, h, t0, s.scale);
    {
        float acc[TMB][NJ];
        zero_acc(acc);
        tok_times_stateT<MSZ>(acc, sS, K, Dst, 0, s, b, h, t0);
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) acc[i][j] *= sfw[ty + 16 * i];
        simt_mm<TMB, NJ>(acc, CB, [&](int t, int r) { return sP[r * LPB + t]; },
                         [&](int r, int i) { return sY1[r * LDM + i]; });
#pragma unroll
        for (int i = 0; i < TMB; ++i)
#pragma unroll
            for (int j = 0; j < NJ; ++j) sDA[(ty + 16 * i) * LDM + tx + 16 * j] += acc[i][j];
    }
    __syncthreads();
    // per token: d beta, d lambda from the write vector, dG
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const size_t BTH = (size_t)s.B * s.T * s.H;
    for (int t = warp; t < CB; t += 8) {
        const float* da = sDA + t * LDM;
        const float* av = sA + t * LDM;
        float db = 0.f;
#pragma unroll
        for (int u = 0; u < G::NE; ++u) db += da[lane + 32 * u] * av[lane + 32 * u];
        db = warp_sum(db);
        const float om = warp_omega_dot<MSZ>(da, av, lane, s.sl); // <da, Omega a>
        if (lane == 0) {
            const size_t gi = tokbase + (size_t)t * s.H;
            a.tok[2 * BTH + gi] = sdG[t];
            a.tok[3 * BTH + gi] = -om;
            a.tok[4 * BTH + gi] = db / sbeta[t];
        }
    }
}

// ---------------------------------------------------------------------------------------
// Reverse cumulative sums over tokens (fp64) and the activation derivatives.
__device__ __forceinline__ double warp_sum_d(double x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__global__ void __launch_bounds__(256) gate_partial_kernel(BwdArgs a, int nseg) {
    const Shape s = a.s;
    const int seg = blockIdx.x, bh = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int t0 = seg * PREP_SEG, len = min(PREP_SEG, s.T - t0);
    const size_t BTH = (size_t)s.B * s.T * s.H;
    double sg = 0.0, sl = 0.0;
    for (int i = threadIdx.x; i < len; i += blockDim.x) {
        const size_t gi = ((size_t)b * s.T + t0 + i) * s.H + h;
        sg += (double)a.tok[gi] + (double)a.tok[2 * BTH + gi];
        sl += (double)a.tok[BTH + gi] + (double)a.tok[3 * BTH + gi];
    }
    __shared__ double red[2][8];
    sg = warp_sum_d(sg);
    sl = warp_sum_d(sl);
    if ((threadIdx.x & 31) == 0) {
        red[0][threadIdx.x >> 5] = sg;
        red[1][threadIdx.x >> 5] = sl;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double x = 0.0, y = 0.0;
        for (int w = 0; w < 8; ++w) {
            x += red[0][w];
            y += red[1][w];
        }
        const size_t BHn = (size_t)s.B * s.H * nseg;
        a.seg[(size_t)bh * nseg + seg] = x;
        a.seg[BHn + (size_t)bh * nseg + seg] = y;
    }
}

__global__ void __launch_bounds__(256) gate_scan_kernel(BwdArgs a, int nseg) {
    const Shape s = a.s;
    const int seg = blockIdx.x, bh = blockIdx.y, b = bh / s.H, h = bh % s.H;
    const int t0 = seg * PREP_SEG, len = min(PREP_SEG, s.T - t0);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const size_t BTH = (size_t)s.B * s.T * s.H;
    const size_t BHn = (size_t)s.B * s.H * nseg;
    __shared__ double s_base[2], s_wt[2][8], s_red[8];
    if (warp == 0) {
        double x = 0.0, y = 0.0;
        for (int k = seg + 1 + lane; k < nseg; k += 32) {
            x += a.seg[(size_t)bh * nseg + k];
            y += a.seg[BHn + (size_t)bh * nseg + k];
        }
        x = warp_sum_d(x);
        y = warp_sum_d(y);
        if (lane == 0) {
            s_base[0] = x;
            s_base[1] = y;
        }
    }
    double xg[4], xl[4], tg = 0.0, tl = 0.0;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int i = 4 * threadIdx.x + u;
        xg[u] = xl[u] = 0.0;
        if (i < len) {
            const size_t gi = ((size_t)b * s.T + t0 + i) * s.H + h;
            xg[u] = (double)a.tok[gi] + (double)a.tok[2 * BTH + gi];
            xl[u] = (double)a.tok[BTH + gi] + (double)a.tok[3 * BTH + gi];
        }
        tg += xg[u];
        tl += xl[u];
    }
    double ig = tg, il = tl;     // inclusive prefix over lanes
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const double yg = __shfl_up_sync(0xffffffffu, ig, o);
        const double yl = __shfl_up_sync(0xffffffffu, il, o);
        if (lane >= o) {
            ig += yg;
            il += yl;
        }
    }
    const double wg = __shfl_sync(0xffffffffu, ig, 31), wl = __shfl_sync(0xffffffffu, il, 31);
    if (lane == 0) {
        s_wt[0][warp] = wg;
        s_wt[1][warp] = wl;
    }
    __syncthreads();
    double later_g = s_base[0] + (wg - ig), later_l = s_base[1] + (wl - il);
    for (int w = warp + 1; w < 8; ++w) {
        later_g += s_wt[0][w];
        later_l += s_wt[1][w];
    }
    const float Ah = a.A[h];
    double dA_acc = 0.0;
    double rg = later_g, rl = later_l;
#pragma unroll
    for (int u = 3; u >= 0; --u) {
        const int i = 4 * threadIdx.x + u;
        rg += xg[u];
        rl += xl[u];
        if (i < len) {
            const size_t gi = ((size_t)b * s.T + t0 + i) * s.H + h;
            const float f = a.decay_logit[gi];
            const float dlogalpha = (float)rg;
            a.d_decay[gi] = dlogalpha * (-Ah * sigmoidf_(f));
            dA_acc += (double)dlogalpha * (double)(-softplusf_(f));
            if (a.d_clock) {   // no clock logits (fixed-rate clock): no clock gradient
                const float delta = sigmoidf_(a.clock_logit[gi]);
                a.d_clock[gi] = (float)rl * delta * (1.f - delta);
            }
            const float bt = a.beta[gi];
            a.d_beta[gi] = a.tok[4 * BTH + gi] * bt * (1.f - bt);
        }
    }
    dA_acc = warp_sum_d(dA_acc);
    if (lane == 0) s_red[warp] = dA_acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < 8; ++w) t += s_red[w];
        a.dA_part[(size_t)bh * nseg + seg] = t;
    }
}

__global__ void dA_final_kernel(BwdArgs a, int nseg) {
    const int h = blockIdx.x * blockDim.x + threadIdx.x;
    if (h >= a.s.H) return;
    double t = 0.0;
    for (int b = 0; b < a.s.B; ++b)
        for (int k = 0; k < nseg; ++k) t += a.dA_part[((size_t)b * a.s.H + h) * nseg + k];
    a.dA[h] = (float)t;
}

// Partial dM over one range of tokens: dMp[h][sp][i][j] = sum over the sp-th of nsplit equal
// ranges of the head's B*T tokens of dl[i] z[j] + p[i] dy[j] (paper order; the per-token vectors
// are [B*H][T][ms] fp32).  Block (i tile, j tile, h * nsplit + sp) forms a 64 x 64 tile of dM
// with 16 x 16 threads holding 4 x 4 outputs each; 32 tokens at a time are staged in shared
// memory (zero past the range's end).
constexpr int DM_TILE = 64, DM_TOK = 32;
__global__ void __launch_bounds__(256) dm_partial_simt(BwdArgs a, int nsplit) {
    const Shape s = a.s;
    const int ms = s.sl.ms;
    const int i0 = blockIdx.x * DM_TILE, j0 = blockIdx.y * DM_TILE;
    const int h = blockIdx.z / nsplit, sp = blockIdx.z % nsplit;
    const long long N = (long long)s.B * s.T;
    const long long n0 = N * sp / nsplit, n1 = N * (sp + 1) / nsplit;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    __shared__ float sL[DM_TOK][DM_TILE], sP[DM_TOK][DM_TILE], sZ[DM_TOK][DM_TILE],
        sY[DM_TOK][DM_TILE];
    float acc[4][4];
    zero_acc(acc);
    for (long long nb = n0; nb < n1; nb += DM_TOK) {
        __syncthreads();
        for (int e = tid; e < DM_TOK * DM_TILE; e += 256) {
            const int r = e / DM_TILE, c = e % DM_TILE;
            const long long n = nb + r;
            float l = 0.f, p = 0.f, z = 0.f, y = 0.f;
            if (n < n1) {
                const long long b = n / s.T, t = n - b * s.T;
                const size_t o = (((size_t)b * s.H + h) * s.T + t) * ms;
                l = a.mDL[o + i0 + c];
                p = a.mP[o + i0 + c];
                z = a.mZ[o + j0 + c];
                y = a.mDY[o + j0 + c];
            }
            sL[r][c] = l;
            sP[r][c] = p;
            sZ[r][c] = z;
            sY[r][c] = y;
        }
        __syncthreads();
#pragma unroll 4
        for (int k = 0; k < DM_TOK; ++k) {
            float l[4], p[4], z[4], y[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                l[u] = sL[k][ty + 16 * u];
                p[u] = sP[k][ty + 16 * u];
                z[u] = sZ[k][tx + 16 * u];
                y[u] = sY[k][tx + 16 * u];
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(l[i], z[j], fmaf(p[i], y[j], acc[i][j]));
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j)
            a.dM[(((size_t)h * nsplit + sp) * ms + i0 + ty + 16 * i) * ms + j0 + tx + 16 * j] =
                acc[i][j];
}

// dR[h][i][k] = sum_j dM[h][i][j] Phi[k][j] for the m active slots i, k (App. A.1
// Eq. app-real-fourier: Phi[k][0] = 1/sqrt(m), Phi[k][2j-1] = sqrt(2/m) cos(2 pi j k / m),
// Phi[k][2j] = sqrt(2/m) sin(2 pi j k / m)); dM is the sum over nsplit partial blocks
// [H][nsplit][ms][ms] in the paper's order (summed in split order).  Block (h, i) of ms threads.
__global__ void __launch_bounds__(MS_MAX) dr_finalize_simt(const float* dMp, int nsplit, float* dR,
                                                           Slots sl) {
    const int h = blockIdx.x, i = blockIdx.y, t = threadIdx.x;
    const int m = sl.m, ms = sl.ms;
    __shared__ float s_dm[MS_MAX], s_ct[MS_MAX], s_st[MS_MAX];
    {
        float acc = 0.f;
        const float* src = dMp + ((size_t)h * nsplit * ms + i) * ms + t;
        for (int sp = 0; sp < nsplit; ++sp) acc += src[(size_t)sp * ms * ms];
        s_dm[t] = acc;
    }
    if (t < m) {
        float sv, cv;
        sincospif((float)t * sl.two_over_m, &sv, &cv);
        s_ct[t] = cv;
        s_st[t] = sv;
    }
    __syncthreads();
    if (t < m) {
        float ac = 0.f, as = 0.f;
        int idx = 0;   // (j t) mod m
        for (int j = 1; j <= sl.npair; ++j) {
            idx += t;
            if (idx >= m) idx -= m;
            ac = fmaf(s_dm[2 * j - 1], s_ct[idx], ac);
            as = fmaf(s_dm[2 * j], s_st[idx], as);
        }
        dR[((size_t)h * m + i) * m + t] = s_dm[0] * sl.inv_sqrt_m + sl.sqrt2_over_m * (ac + as);
    }
}

template <int D, int MSZ, typename TI>
cudaError_t bwd_dispatch(const BwdArgs& a, cudaStream_t st) {
    using G = Geo<MSZ>;
    constexpr int CB = G::CB, LDM = G::LDM;
    const Shape& s = a.s;
    FwdArgs f{};
    f.s = s;
    f.q = a.q;
    f.k = a.k;
    f.v = a.v;
    f.lam = a.lam;
    f.g = a.g;
    f.beta = a.beta;
    f.states = a.states;
    cudaError_t e = a.states_given ? cudaSuccess : launch_state_simt(f, st);
    if (e != cudaSuccess) return e;
    const dim3 gchunk(s.nchunk(), s.B * s.H);
    constexpr int SSZ = staging_floats<D, MSZ>();
    const size_t sm1 = (size_t)(4 * CB * LDM + SSZ + CB * G::LPB + 6 * CB + 32 * LDM) * sizeof(float);
    auto k1 = bwd_intra1_kernel<D, MSZ, TI>;
    cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm1);
    { LaunchScope ls_("bwd_intra1", st); k1<<<gchunk, 256, sm1, st>>>(a); }
    const size_t sma = (size_t)(CB * LDM + CB * 65 + CB) * sizeof(float);
    auto ka = adj_state_kernel<MSZ, TI>;
    cudaFuncSetAttribute(ka, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sma);
    { LaunchScope ls_("bwd_adjoint", st); ka<<<dim3(2 * D / 64, s.B * s.H, MSZ / 128), 256, sma, st>>>(a); }
    const size_t sm2 = (size_t)(4 * CB * LDM + SSZ + CB * G::LPB + 5 * CB) * sizeof(float);
    auto k2 = bwd_intra2_kernel<D, MSZ, TI>;
    cudaFuncSetAttribute(k2, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm2);
    { LaunchScope ls_("bwd_intra2", st); k2<<<gchunk, 256, sm2, st>>>(a); }
    if (a.dR) {
        const int ns = dm_splits(s);
        const dim3 gdm(MSZ / DM_TILE, MSZ / DM_TILE, s.H * ns);
        { LaunchScope ls_("bwd_dm_reduce", st); dm_partial_simt<<<gdm, 256, 0, st>>>(a, ns); }
        { LaunchScope ls_("bwd_dr_finalize", st); dr_finalize_simt<<<dim3(s.H, s.sl.m), MSZ, 0, st>>>(a.dM, ns, a.dR, s.sl); }
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return launch_bwd_gates(a, st);
}

template <int MSZ>
cudaError_t bwd_dispatch_d(const BwdArgs& a, cudaStream_t st) {
    const Shape& s = a.s;
    if (s.D == 128) return s.bf16 ? bwd_dispatch<128, MSZ, __nv_bfloat16>(a, st) : bwd_dispatch<128, MSZ, float>(a, st);
    if (s.D == 64) return s.bf16 ? bwd_dispatch<64, MSZ, __nv_bfloat16>(a, st) : bwd_dispatch<64, MSZ, float>(a, st);
    if (s.D == 256) return s.bf16 ? bwd_dispatch<256, MSZ, __nv_bfloat16>(a, st) : bwd_dispatch<256, MSZ, float>(a, st);
    return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t simt_bwd_read_error(cudaStream_t st, int* err) { return read_simt_error(st, err); }

cudaError_t launch_bwd_gates(const BwdArgs& a, cudaStream_t st) {
    const Shape& s = a.s;
    const int nseg = (s.T + PREP_SEG - 1) / PREP_SEG;
    { LaunchScope ls_("bwd_gate_partial", st); gate_partial_kernel<<<dim3(nseg, s.B * s.H), 256, 0, st>>>(a, nseg); }
    { LaunchScope ls_("bwd_gate_scan", st); gate_scan_kernel<<<dim3(nseg, s.B * s.H), 256, 0, st>>>(a, nseg); }
    if (a.dA) { LaunchScope ls_("bwd_dA", st); dA_final_kernel<<<(s.H + 127) / 128, 128, 0, st>>>(a, nseg); }
    return cudaGetLastError();
}

cudaError_t launch_bwd_simt(const BwdArgs& a, cudaStream_t st) {
    const Shape& s = a.s;
    if (s.C != bwd_chunk(s.sl)) return cudaErrorInvalidValue;
    if (s.sl.ms == 128) return bwd_dispatch_d<128>(a, st);
    if (s.sl.ms == 256) return bwd_dispatch_d<256>(a, st);
    return cudaErrorInvalidValue;
}

}  // namespace cyfa
