// cyfa_step: one decode token against the persistent fp32 states (Sec. 3.2 Eq.
// cyfa-absolute-recurrence and Eq. cyfa-absolute-readout applied to a single token).
//
// The step is HBM-bound: per (b, h) it streams the fp32 Kbar and Vbar (64 KiB each at d = 128)
// in and out once.  d = 128 runs a persistent, warp-specialised pipeline (step_pipe_kernel): one
// block per SM walks a contiguous, head-major range of (b, h) rows; the key stream of one row,
// the middle readout of the previous row and the value stream of the row before run at once, so
// the HBM streams are never idle during the readout arithmetic; the state rows arrive through a
// two-stage cp.async ring per streaming warp.  Other d and m run the simpler step_kernel (G batch rows
// of one head per 256-thread block).  The middle readout applies Phi through an m-entry cosine /
// sine table (entry (j r) mod m of Eq. app-real-fourier) and R; m > 127 keeps 256 storage rows.
#include "common.cuh"
#include "kernels.h"

namespace cyfa {

namespace {

constexpr int G = 4;          // batch rows per block
constexpr int BATCH = 8;      // rows loaded per warp before they are used

// A lane's VPL consecutive floats of a state row (VPL = 2, 4 or 8), by 8- or 16-byte accesses.
template <int VPL>
__device__ __forceinline__ void load_row(float (&x)[VPL], const float* p) {
    if constexpr (VPL == 2) {
        const float2 t = *reinterpret_cast<const float2*>(p);
        x[0] = t.x; x[1] = t.y;
    } else {
#pragma unroll
        for (int u = 0; u < VPL; u += 4) {
            const float4 t = *reinterpret_cast<const float4*>(p + u);
            x[u] = t.x; x[u + 1] = t.y; x[u + 2] = t.z; x[u + 3] = t.w;
        }
    }
}
template <int VPL>
__device__ __forceinline__ void store_row(float* p, const float (&x)[VPL]) {
    if constexpr (VPL == 2) {
        *reinterpret_cast<float2*>(p) = make_float2(x[0], x[1]);
    } else {
#pragma unroll
        for (int u = 0; u < VPL; u += 4)
            *reinterpret_cast<float4*>(p + u) = make_float4(x[u], x[u + 1], x[u + 2], x[u + 3]);
    }
}

// Generic step for MSZ storage rows (128 for m <= 127, 256 above); G batch rows of one head per
// 256-thread block.
template <int D, int MSZ, typename TI>
__global__ void __launch_bounds__(256) step_kernel(StepArgs a) {
    constexpr int VPL = D / 32;   // floats per lane per state row
    constexpr int HP = MSZ / 2;   // entry pairs of a slot vector (the DC / padding pair is j = 0)
    const int h = blockIdx.y, b0 = blockIdx.x * G;
    const int ng = min(G, a.B - b0);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const Slots sl = a.sl;
    const int m = sl.m;
    __shared__ float s_ct[MSZ - 1], s_st[MSZ - 1];
    // q and k, then (after the key pass has taken them into registers) the two halves of o
    __shared__ float s_qk[2][G][D];
    __shared__ float s_v[G][D];
    __shared__ float s_a[G][MSZ], s_o1[G][MSZ], s_z[G][MSZ], s_u[G][MSZ], s_l[G][MSZ], s_y[G][MSZ];
    __shared__ float s_cs[G][HP], s_sn[G][HP];
    __shared__ float s_alpha[G], s_inv[G];
    __shared__ double s_lam[G];
    float (*s_q)[D] = s_qk[0];
    float (*s_k)[D] = s_qk[1];
    float (*s_opart)[G][D] = s_qk;

    const TI* Q = (const TI*)a.q;
    const TI* K = (const TI*)a.k;
    const TI* V = (const TI*)a.v;
    if (tid < m) {
        float s, c;
        sincospif((float)tid * sl.two_over_m, &s, &c);
        s_ct[tid] = c;
        s_st[tid] = s;
    }
    for (int e = tid; e < G * D; e += 256) {
        const int g = e / D, i = e % D;
        if (g < ng) {
            const size_t bh = (size_t)(b0 + g) * a.H + h;
            s_q[g][i] = a.scale * ldf(Q, bh * D + i);
            s_k[g][i] = ldf(K, bh * D + i);
            s_v[g][i] = ldf(V, bh * D + i);
        }
    }
    // clock, gates and rotation angles: (g, j) with j = 0 for the DC entry
    for (int e = tid; e < G * HP; e += 256) {
        const int g = e / HP, j = e % HP;
        if (g < ng) {
            const size_t bh = (size_t)(b0 + g) * a.H + h;
            const double lam_new = a.lambda[bh] + (double)sigmoidf_(a.clock_logit[bh]);
            const float lam = (float)(lam_new - (double)m * floor(lam_new / (double)m));
            const float beta = sigmoidf_(a.beta_logit[bh]);
            if (j == 0) {
                s_alpha[g] = expf(-a.A[h] * softplusf_(a.decay_logit[bh]));
                s_lam[g] = lam_new;
                s_a[g][0] = beta * sl.inv_sqrt_m;
                s_a[g][MSZ - 1] = 0.f;
                s_cs[g][0] = 1.f;
                s_sn[g][0] = 0.f;
            } else if (j <= sl.npair) {
                float s, c;
                sincospif(phase_pi_m(lam, j, sl), &s, &c);
                s_cs[g][j] = c;
                s_sn[g][j] = s;
                s_a[g][2 * j - 1] = beta * sl.sqrt2_over_m * c;
                s_a[g][2 * j] = -beta * sl.sqrt2_over_m * s;
            } else {   // padding slots: no write, no rotation
                s_cs[g][j] = 1.f;
                s_sn[g][j] = 0.f;
                s_a[g][2 * j - 1] = 0.f;
                s_a[g][2 * j] = 0.f;
            }
        }
    }
    __syncthreads();

    // Kbar <- alpha Kbar + a k^T ; o' = Kbar (s q).  Warps 2g and 2g+1 own batch row g; warp
    // (2g + half) owns state rows r = half + 2 i.
    const int wg = warp >> 1, half = warp & 1;
    if (wg < ng) {
        const int g = wg;
        float* Kb = a.Kbar + ((size_t)(b0 + g) * a.H + h) * MSZ * D;
        const float alpha = s_alpha[g];
        float qv[VPL], kv[VPL];
#pragma unroll
        for (int u = 0; u < VPL; ++u) {
            qv[u] = s_q[g][lane * VPL + u];
            kv[u] = s_k[g][lane * VPL + u];
        }
        for (int i0 = 0; i0 < MSZ / 2; i0 += BATCH) {
            float x[BATCH][VPL];
#pragma unroll
            for (int bb = 0; bb < BATCH; ++bb) {
                const int r = half + 2 * (i0 + bb);
                load_row<VPL>(x[bb], Kb + r * D + lane * VPL);
            }
#pragma unroll
            for (int bb = 0; bb < BATCH; ++bb) {
                const int r = half + 2 * (i0 + bb);
                const float ar = s_a[g][r];
                float dot = 0.f;
#pragma unroll
                for (int u = 0; u < VPL; ++u) {
                    x[bb][u] = fmaf(alpha, x[bb][u], ar * kv[u]);
                    dot = fmaf(x[bb][u], qv[u], dot);
                }
                store_row<VPL>(Kb + r * D + lane * VPL, x[bb]);
                dot = warp_sum(dot);
                if (lane == 0) s_o1[g][r] = dot;
            }
        }
    }
    __syncthreads();

    // middle readout (Sec. 3.3 Eq. cyfa-two-pass, middle line) for the G rows:
    // z = U(lam) o'; u = Phi z; l = R u; p = softmax(l); y' = R^T p; y = Phi^T y'; o'' = U(-lam) y
    for (int e = tid; e < G * HP; e += 256) {
        const int g = e / HP, j = e % HP;
        if (g < ng) {
            if (j == 0) {
                s_z[g][0] = s_o1[g][0];
                s_z[g][MSZ - 1] = 0.f;
            } else {   // padding pairs have c = 1, sn = 0 and zero entries
                const float c = s_cs[g][j], sn = s_sn[g][j];
                const float xc = s_o1[g][2 * j - 1], xs = s_o1[g][2 * j];
                s_z[g][2 * j - 1] = c * xc - sn * xs;
                s_z[g][2 * j] = sn * xc + c * xs;
            }
        }
    }
    __syncthreads();
    for (int e = tid; e < G * MSZ; e += 256) {   // u_r = z_0/sqrt(m) + sqrt(2/m) sum_j (...)
        const int g = e / MSZ, r = e % MSZ;
        if (g < ng && r < m) {
            float acc = 0.f;
            int idx = 0;
            for (int j = 1; j <= sl.npair; ++j) {
                idx += r;
                if (idx >= m) idx -= m;
                acc = fmaf(s_z[g][2 * j - 1], s_ct[idx], acc);
                acc = fmaf(s_z[g][2 * j], s_st[idx], acc);
            }
            s_u[g][r] = s_z[g][0] * sl.inv_sqrt_m + sl.sqrt2_over_m * acc;
        }
    }
    __syncthreads();
    const float* Rh = a.R + (size_t)h * m * m;
    for (int i = warp; i < m; i += 8) {   // l_i = sum_r R[i][r] u_r, one R row per warp
        constexpr int NE = MSZ / 32;
        float rv[NE];
#pragma unroll
        for (int k = 0; k < NE; ++k) {
            const int r = lane + 32 * k;
            rv[k] = r < m ? Rh[i * m + r] : 0.f;
        }
        for (int g = 0; g < ng; ++g) {
            float acc = 0.f;
#pragma unroll
            for (int k = 0; k < NE; ++k) {
                const int r = lane + 32 * k;
                if (r < m) acc = fmaf(rv[k], s_u[g][r], acc);
            }
            acc = warp_sum(acc);
            if (lane == 0) s_l[g][i] = acc;
        }
    }
    __syncthreads();
    if (warp < ng) {
        const int g = warp;
        float mx = -INFINITY;
        for (int i = lane; i < m; i += 32) mx = fmaxf(mx, s_l[g][i]);
        mx = warp_max(mx);
        float sum = 0.f;
        for (int i = lane; i < m; i += 32) {
            const float e = expf(s_l[g][i] - mx);
            s_l[g][i] = e;
            sum += e;
        }
        sum = warp_sum(sum);
        if (lane == 0) s_inv[g] = 1.f / sum;
    }
    __syncthreads();
    // y'_r = sum_i R[i][r] p_i, thread (r mod 128, half): rows g = half, half + 2
    for (int r = tid & 127; r < m; r += 128) {
        const int g0 = tid >> 7, g1 = g0 + 2;
        float acc0 = 0.f, acc1 = 0.f;
        for (int i = 0; i < m; ++i) {
            const float rv = Rh[i * m + r];
            acc0 = fmaf(rv, s_l[g0][i], acc0);
            acc1 = fmaf(rv, s_l[g1][i], acc1);
        }
        if (g0 < ng) s_u[g0][r] = acc0 * s_inv[g0];
        if (g1 < ng) s_u[g1][r] = acc1 * s_inv[g1];
    }
    __syncthreads();
    for (int e = tid; e < G * HP; e += 256) {   // y = Phi^T y', then o'' = U(-lam) y on (2j-1, 2j)
        const int g = e / HP, j = e % HP;
        if (g < ng) {
            if (j == 0) {
                float ac = 0.f;
                for (int r = 0; r < m; ++r) ac += s_u[g][r];
                s_y[g][0] = ac * sl.inv_sqrt_m;
                s_y[g][MSZ - 1] = 0.f;
            } else if (j > sl.npair) {   // padding slots
                s_y[g][2 * j - 1] = 0.f;
                s_y[g][2 * j] = 0.f;
            } else {
                float ac = 0.f, as = 0.f;
                int idx = 0;
                for (int r = 0; r < m; ++r) {
                    ac = fmaf(s_u[g][r], s_ct[idx], ac);
                    as = fmaf(s_u[g][r], s_st[idx], as);
                    idx += j;
                    if (idx >= m) idx -= m;
                }
                const float yc = sl.sqrt2_over_m * ac, ys = sl.sqrt2_over_m * as;
                const float c = s_cs[g][j], sn = s_sn[g][j];
                s_y[g][2 * j - 1] = c * yc + sn * ys;
                s_y[g][2 * j] = -sn * yc + c * ys;
            }
        }
    }
    __syncthreads();

    // Vbar <- alpha Vbar + a v^T ; o = Vbar^T o''
    if (wg < ng) {
        const int g = wg;
        float* Vb = a.Vbar + ((size_t)(b0 + g) * a.H + h) * MSZ * D;
        const float alpha = s_alpha[g];
        float vv[VPL], oacc[VPL];
#pragma unroll
        for (int u = 0; u < VPL; ++u) {
            vv[u] = s_v[g][lane * VPL + u];
            oacc[u] = 0.f;
        }
        for (int i0 = 0; i0 < MSZ / 2; i0 += BATCH) {
            float x[BATCH][VPL];
#pragma unroll
            for (int bb = 0; bb < BATCH; ++bb) {
                const int r = half + 2 * (i0 + bb);
                load_row<VPL>(x[bb], Vb + r * D + lane * VPL);
            }
#pragma unroll
            for (int bb = 0; bb < BATCH; ++bb) {
                const int r = half + 2 * (i0 + bb);
                const float ar = s_a[g][r], yr = s_y[g][r];
#pragma unroll
                for (int u = 0; u < VPL; ++u) {
                    x[bb][u] = fmaf(alpha, x[bb][u], ar * vv[u]);
                    oacc[u] = fmaf(x[bb][u], yr, oacc[u]);
                }
                store_row<VPL>(Vb + r * D + lane * VPL, x[bb]);
            }
        }
#pragma unroll
        for (int u = 0; u < VPL; ++u) s_opart[half][g][lane * VPL + u] = oacc[u];
    }
    __syncthreads();
    for (int e = tid; e < ng * D; e += 256) {
        const int g = e / D, i = e % D;
        stf((TI*)a.o, ((size_t)(b0 + g) * a.H + h) * D + i, s_opart[0][g][i] + s_opart[1][g][i]);
    }
    if (tid < ng) a.lambda[(size_t)(b0 + tid) * a.H + h] = s_lam[tid];
}

// ---------------------------------------------------------------------------------------
// d = 128: persistent, warp-specialised pipeline over (b, h) rows.  Each block owns a
// contiguous range of rows ordered head-major (so R of a head is loaded into shared memory once
// per block and head) and runs three warp groups on consecutive rows at once:
//   warps 0-7   key stream of row i     (gates, write vector, Kbar <- alpha Kbar + a k^T, o')
//   warps 16-19 middle readout of row i-1 (o' -> o'', all in shared memory)
//   warps 8-15  value stream of row i-2  (Vbar <- alpha Vbar + a v^T, o = Vbar^T o'')
// so the HBM streams of two rows overlap the readout arithmetic of a third.  Per-row vectors
// live in a three-slot ring; one block barrier closes every step of the pipeline.
constexpr int PK_W = 8, PV_W = 8, PM_W = 4;
constexpr int P_THREADS = (PK_W + PV_W + PM_W) * 32;
constexpr int P_RING = 3;
constexpr int P_BATCH = 8;

struct PipeSlot {
    float a[MS];          // write vector beta U(-lam) b
    float cs[64], sn[64]; // cos / sin of the pair angles (entry 0: 1, 0)
    float q[128], k[128], v[128];
    float o1[MS];         // o'
    float o2[MS];         // o''
    float alpha;
    int bh;
};
struct PipeSmem {
    float stage[PK_W + PV_W][2][P_BATCH][128];   // cp.async ring of state rows, per streaming warp
    float R[MA * MA];
    float ct[MA], st[MA];
    float z[MS], u[MS], l[MS], red[2][8];
    float vred[PV_W][128];
    PipeSlot slot[P_RING];
    int head;
};

__device__ __forceinline__ void named_bar(int id, int n) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}
// Eight consecutive 512-byte state rows (a warp's batch) global -> shared, 16 bytes per lane per
// row, asynchronously; one commit group per batch.
__device__ __forceinline__ void prefetch_rows(float* dst, const float* src, int lane) {
#pragma unroll
    for (int rr = 0; rr < P_BATCH; ++rr) {
        const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst + rr * 128 + lane * 4));
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d),
                     "l"(src + rr * 128 + lane * 4)
                     : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
}
// R of head h (127 x 127 fp32) global -> shared with 4-byte asynchronous copies (rows of R are not
// 16-byte aligned), issued by `nthr` threads; one commit group.
__device__ __forceinline__ void load_R_async(float* dst, const float* R, int h, int t, int nthr) {
    const float* src = R + (size_t)h * MA * MA;
    for (int e = t; e < MA * MA; e += nthr) {
        const uint32_t d = static_cast<uint32_t>(__cvta_generic_to_shared(dst + e));
        asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(d), "l"(src + e) : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void wait_prefetch_but_one() {
    asm volatile("cp.async.wait_group 1;" ::: "memory");
}
__device__ __forceinline__ void wait_prefetch_all() {
    asm volatile("cp.async.wait_group 0;" ::: "memory");
}

template <typename TI>
__global__ void __launch_bounds__(P_THREADS, 1) step_pipe_kernel(StepArgs a) {
    constexpr int D = 128;
    extern __shared__ __align__(16) uint8_t pipe_raw[];
    PipeSmem& S = *reinterpret_cast<PipeSmem*>(pipe_raw);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int NR = a.B * a.H;
    const int w0 = (int)((long long)NR * blockIdx.x / gridDim.x);
    const int w1 = (int)((long long)NR * (blockIdx.x + 1) / gridDim.x);
    const int n = w1 - w0;
    const TI* Q = (const TI*)a.q;
    const TI* K = (const TI*)a.k;
    const TI* V = (const TI*)a.v;
    if (tid < MA) {
        float sv, cv;
        sincospif((float)tid * (2.f / 127.f), &sv, &cv);
        S.ct[tid] = cv;
        S.st[tid] = sv;
    }
    // R of the first row's head, loaded by the whole block before the pipeline starts
    if (n > 0) {
        load_R_async(S.R, a.R, w0 / a.B, tid, P_THREADS);
        asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    if (tid == 0) S.head = n > 0 ? w0 / a.B : -1;
    auto bh_of = [&](int i) {   // (b, h) index of the block's i-th row
        const int w = w0 + i, hh = w / a.B;
        return (w - hh * a.B) * a.H + hh;
    };
    // each streaming warp owns 16 consecutive state rows, two batches of 8; batch g of the warp's
    // sequence (row g / 2, half g % 2) sits in stage g % 2, and batch g + 1 is in flight while g
    // is used
    const bool kwarp = warp < PK_W, vwarp = warp >= PK_W && warp < PK_W + PV_W;
    const int sw = kwarp ? warp : warp - PK_W;
    if ((kwarp || vwarp) && n > 0) {
        const float* base = (kwarp ? a.Kbar : a.Vbar) + (size_t)bh_of(0) * MS * 128;
        prefetch_rows(&S.stage[warp][0][0][0], base + (size_t)(16 * sw) * 128, lane);
    }
    __syncthreads();
    for (int it = 0; it < n + 2; ++it) {
        if (warp < PK_W) {
            // ------------------------------------------------------------ key stream, row it
            if (it < n) {
                const int w = w0 + it, h = w / a.B, b = w - h * a.B;
                const int bh = b * a.H + h;
                PipeSlot& P = S.slot[it % P_RING];
                const int t = tid;   // 0..255
                if (t < 64) {
                    const int j = t;
                    const double lam_new = a.lambda[bh] + (double)sigmoidf_(a.clock_logit[bh]);
                    const float lam = (float)(lam_new - 127.0 * floor(lam_new / 127.0));
                    const float beta = sigmoidf_(a.beta_logit[bh]);
                    if (j == 0) {
                        P.alpha = expf(-a.A[h] * softplusf_(a.decay_logit[bh]));
                        P.bh = bh;
                        P.a[0] = beta * INV_SQRT_M;
                        P.a[127] = 0.f;
                        P.cs[0] = 1.f;
                        P.sn[0] = 0.f;
                    } else {
                        float sv, cv;
                        sincospif(phase_pi(lam, j), &sv, &cv);
                        P.cs[j] = cv;
                        P.sn[j] = sv;
                        P.a[2 * j - 1] = beta * SQRT_2_OVER_M * cv;
                        P.a[2 * j] = -beta * SQRT_2_OVER_M * sv;
                    }
                    named_bar(1, PK_W * 32);   // every lane has read lambda before it is replaced
                    if (j == 0) a.lambda[bh] = lam_new;
                } else {
                    const int e = t - 64;   // 0..191: q, k, v element pairs
                    for (int i = e; i < 3 * D; i += 192) {
                        const int which = i / D, c = i - which * D;
                        const TI* src = which == 0 ? Q : (which == 1 ? K : V);
                        const float x = ldf(src, (size_t)bh * D + c);
                        if (which == 0) P.q[c] = a.scale * x;
                        else if (which == 1) P.k[c] = x;
                        else P.v[c] = x;
                    }
                    named_bar(1, PK_W * 32);
                }
                named_bar(1, PK_W * 32);   // slot written
                float* Kb = a.Kbar + (size_t)bh * MS * D;
                const float alpha = P.alpha;
                float qv[4], kv[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    qv[u] = P.q[lane * 4 + u];
                    kv[u] = P.k[lane * 4 + u];
                }
#pragma unroll 1
                for (int half = 0; half < 2; ++half) {
                    // next batch in flight: this row's second half, or the next row's first
                    if (half == 0) {
                        prefetch_rows(&S.stage[warp][1][0][0], Kb + (size_t)(16 * sw + 8) * D, lane);
                    } else if (it + 1 < n) {
                        prefetch_rows(&S.stage[warp][0][0][0],
                                      a.Kbar + (size_t)bh_of(it + 1) * MS * D + (size_t)(16 * sw) * D, lane);
                    } else {
                        asm volatile("cp.async.commit_group;" ::: "memory");
                    }
                    wait_prefetch_but_one();
                    __syncwarp();
                    const float* stg = &S.stage[warp][half][0][0];
#pragma unroll
                    for (int bb = 0; bb < P_BATCH; ++bb) {
                        const int r = 16 * sw + 8 * half + bb;
                        const float4 f = *reinterpret_cast<const float4*>(stg + bb * 128 + lane * 4);
                        float x[4] = {f.x, f.y, f.z, f.w};
                        const float ar = P.a[r];
                        float dot = 0.f;
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            x[u] = fmaf(alpha, x[u], ar * kv[u]);
                            dot = fmaf(x[u], qv[u], dot);
                        }
                        *reinterpret_cast<float4*>(Kb + r * D + lane * 4) = make_float4(x[0], x[1], x[2], x[3]);
                        dot = warp_sum(dot);
                        if (lane == 0) P.o1[r] = dot;
                    }
                    __syncwarp();   // the stage is read before the next prefetch overwrites it
                }
            }
        } else if (warp < PK_W + PV_W) {
            // ---------------------------------------------------------- value stream, row it-2
            if (it >= 2) {
                const int vw = warp - PK_W;
                PipeSlot& P = S.slot[(it - 2) % P_RING];
                const int bh = P.bh;
                float* Vb = a.Vbar + (size_t)bh * MS * D;
                const float alpha = P.alpha;
                float vv[4], oacc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int u = 0; u < 4; ++u) vv[u] = P.v[lane * 4 + u];
                const int vrow = it - 2;   // the block's row index of this value stream
#pragma unroll 1
                for (int half = 0; half < 2; ++half) {
                    if (half == 0) {
                        prefetch_rows(&S.stage[warp][1][0][0], Vb + (size_t)(16 * vw + 8) * D, lane);
                    } else if (vrow + 1 < n) {
                        prefetch_rows(&S.stage[warp][0][0][0],
                                      a.Vbar + (size_t)bh_of(vrow + 1) * MS * D + (size_t)(16 * vw) * D, lane);
                    } else {
                        asm volatile("cp.async.commit_group;" ::: "memory");
                    }
                    wait_prefetch_but_one();
                    __syncwarp();
                    const float* stg = &S.stage[warp][half][0][0];
#pragma unroll
                    for (int bb = 0; bb < P_BATCH; ++bb) {
                        const int r = 16 * vw + 8 * half + bb;
                        const float4 f = *reinterpret_cast<const float4*>(stg + bb * 128 + lane * 4);
                        float x[4] = {f.x, f.y, f.z, f.w};
                        const float ar = P.a[r], yr = P.o2[r];
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            x[u] = fmaf(alpha, x[u], ar * vv[u]);
                            oacc[u] = fmaf(x[u], yr, oacc[u]);
                        }
                        *reinterpret_cast<float4*>(Vb + r * D + lane * 4) = make_float4(x[0], x[1], x[2], x[3]);
                    }
                    __syncwarp();
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) S.vred[vw][lane * 4 + u] = oacc[u];
                named_bar(3, PV_W * 32);
                const int t = tid - PK_W * 32;   // 0..255
                if (t < D) {
                    float o = 0.f;
#pragma unroll
                    for (int w = 0; w < PV_W; ++w) o += S.vred[w][t];
                    stf((TI*)a.o, (size_t)bh * D + t, o);
                }
            }
        } else {
            // --------------------------------------------------------- middle readout, row it-1
            if (it >= 1 && it - 1 < n) {
                const int m = tid - (PK_W + PV_W) * 32;   // 0..127
                const int mw = m >> 5;
                PipeSlot& P = S.slot[(it - 1) % P_RING];
                const int w = w0 + it - 1, h = w / a.B;
                if (h != S.head) {   // a new head: its R (the readout group has no other copies)
                    load_R_async(S.R, a.R, h, m, PM_W * 32);
                    asm volatile("cp.async.wait_group 0;" ::: "memory");
                    named_bar(2, PM_W * 32);
                    if (m == 0) S.head = h;
                }
                // z = U(lam) o'
                if (m < 64) {
                    const int j = m;
                    if (j == 0) {
                        S.z[0] = P.o1[0];
                        S.z[127] = 0.f;
                    } else {
                        const float c = P.cs[j], sn = P.sn[j];
                        const float xc = P.o1[2 * j - 1], xs = P.o1[2 * j];
                        S.z[2 * j - 1] = c * xc - sn * xs;
                        S.z[2 * j] = sn * xc + c * xs;
                    }
                }
                named_bar(2, PM_W * 32);
                // u = Phi z (slot r); four independent chains over the pairs j = 1..63
                if (m < MA) {
                    float acc[4] = {0.f, 0.f, 0.f, 0.f};
                    int idx[4];
                    const int m4 = (4 * m) % MA;
#pragma unroll
                    for (int c = 0; c < 4; ++c) idx[c] = ((c + 1) * m) % MA;
                    for (int j0 = 1; j0 <= NPAIR; j0 += 4) {
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            const int j = j0 + c;
                            if (j <= NPAIR) {
                                acc[c] = fmaf(S.z[2 * j - 1], S.ct[idx[c]], acc[c]);
                                acc[c] = fmaf(S.z[2 * j], S.st[idx[c]], acc[c]);
                            }
                            idx[c] += m4;
                            if (idx[c] >= MA) idx[c] -= MA;
                        }
                    }
                    S.u[m] = S.z[0] * INV_SQRT_M + SQRT_2_OVER_M * ((acc[0] + acc[1]) + (acc[2] + acc[3]));
                }
                named_bar(2, PM_W * 32);
                // l = R u ; softmax over the m active slots
                float lv = -INFINITY;
                if (m < MA) {
                    float acc[4] = {0.f, 0.f, 0.f, 0.f};
                    const float* Rr = S.R + m * MA;
                    for (int c0 = 0; c0 < MA; c0 += 4) {
#pragma unroll
                        for (int c = 0; c < 4; ++c)
                            if (c0 + c < MA) acc[c] = fmaf(Rr[c0 + c], S.u[c0 + c], acc[c]);
                    }
                    lv = (acc[0] + acc[1]) + (acc[2] + acc[3]);
                }
                float mx = warp_max(lv);
                if (lane == 0) S.red[0][mw] = mx;
                named_bar(2, PM_W * 32);
                mx = fmaxf(fmaxf(S.red[0][0], S.red[0][1]), fmaxf(S.red[0][2], S.red[0][3]));
                const float e = (m < MA) ? expf(lv - mx) : 0.f;
                float sum = warp_sum(e);
                if (lane == 0) S.red[1][mw] = sum;
                S.l[m] = e;
                named_bar(2, PM_W * 32);
                const float inv = 1.f / ((S.red[1][0] + S.red[1][1]) + (S.red[1][2] + S.red[1][3]));
                // y'_c = sum_r R[r][c] p_r
                if (m < MA) {
                    float acc[4] = {0.f, 0.f, 0.f, 0.f};
                    for (int r0 = 0; r0 < MA; r0 += 4) {
#pragma unroll
                        for (int c = 0; c < 4; ++c)
                            if (r0 + c < MA) acc[c] = fmaf(S.R[(r0 + c) * MA + m], S.l[r0 + c], acc[c]);
                    }
                    S.u[m] = ((acc[0] + acc[1]) + (acc[2] + acc[3])) * inv;
                }
                named_bar(2, PM_W * 32);
                // y = Phi^T y' ; o'' = U(-lam) y
                if (m < 64) {
                    const int j = m;
                    if (j == 0) {
                        float ac[4] = {0.f, 0.f, 0.f, 0.f};
                        for (int r0 = 0; r0 < MA; r0 += 4) {
#pragma unroll
                            for (int c = 0; c < 4; ++c)
                                if (r0 + c < MA) ac[c] += S.u[r0 + c];
                        }
                        P.o2[0] = ((ac[0] + ac[1]) + (ac[2] + ac[3])) * INV_SQRT_M;
                        P.o2[127] = 0.f;
                    } else {
                        float ac[4] = {0.f, 0.f, 0.f, 0.f}, as[4] = {0.f, 0.f, 0.f, 0.f};
                        int idx[4];
                        const int j4 = (4 * j) % MA;
#pragma unroll
                        for (int c = 0; c < 4; ++c) idx[c] = (c * j) % MA;
                        for (int r0 = 0; r0 < MA; r0 += 4) {
#pragma unroll
                            for (int c = 0; c < 4; ++c) {
                                if (r0 + c < MA) {
                                    ac[c] = fmaf(S.u[r0 + c], S.ct[idx[c]], ac[c]);
                                    as[c] = fmaf(S.u[r0 + c], S.st[idx[c]], as[c]);
                                }
                                idx[c] += j4;
                                if (idx[c] >= MA) idx[c] -= MA;
                            }
                        }
                        const float yc = SQRT_2_OVER_M * ((ac[0] + ac[1]) + (ac[2] + ac[3]));
                        const float ys = SQRT_2_OVER_M * ((as[0] + as[1]) + (as[2] + as[3]));
                        const float c = P.cs[j], sn = P.sn[j];
                        P.o2[2 * j - 1] = c * yc + sn * ys;
                        P.o2[2 * j] = -sn * yc + c * ys;
                    }
                }
            }
        }
        __syncthreads();
    }
    wait_prefetch_all();
}

template <int MSZ>
cudaError_t launch_generic(const StepArgs& a, dim3 grid, cudaStream_t st) {
    LaunchScope ls_("decode_step", st);
#define CYFA_STEP(DD)                                                                   \
    if (a.D == DD) {                                                                    \
        if (a.bf16) step_kernel<DD, MSZ, __nv_bfloat16><<<grid, 256, 0, st>>>(a);       \
        else step_kernel<DD, MSZ, float><<<grid, 256, 0, st>>>(a);                      \
        return cudaGetLastError();                                                      \
    }
    CYFA_STEP(64)
    CYFA_STEP(128)
    CYFA_STEP(256)
#undef CYFA_STEP
    return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_step(const StepArgs& a, cudaStream_t st) {
    const dim3 grid((a.B + G - 1) / G, a.H);
    if (a.D == 128 && a.sl.m == 127) {
        int dev = 0, sms = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return e;
        const int rows = a.B * a.H;
        const int blocks = rows < sms ? rows : sms;
        const int smem = (int)sizeof(PipeSmem);
        if (a.bf16) {
            auto k = step_pipe_kernel<__nv_bfloat16>;
            cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
            LaunchScope ls_("decode_step", st);
            k<<<blocks, P_THREADS, smem, st>>>(a);
        } else {
            auto k = step_pipe_kernel<float>;
            cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
            LaunchScope ls_("decode_step", st);
            k<<<blocks, P_THREADS, smem, st>>>(a);
        }
    } else {   // the generic kernel
        const cudaError_t e = a.sl.ms == 128 ? launch_generic<128>(a, grid, st)
                                             : launch_generic<256>(a, grid, st);
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

}  // namespace cyfa
