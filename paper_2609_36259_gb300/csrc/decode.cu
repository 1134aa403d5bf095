// cyfa_step: one decode token against the persistent fp32 states (Sec. 3.2 Eq.
// cyfa-absolute-recurrence and Eq. cyfa-absolute-readout applied to a single token).
//
// The step is HBM-bound: per (b, h) it streams the fp32 Kbar and Vbar (64 KiB each at d = 128)
// in and out once.  One 256-thread block serves G batch rows of one head, so the readout
// matrix R of the head is read from L2 once per G rows.  Each state is streamed in batches of
// eight 512-byte rows per warp (loads issued before the dependent arithmetic) with 16-byte
// accesses; two warps share each batch row.  The middle readout applies Phi through a 127-entry cosine / sine table (entry
// (j r) mod m of Eq. app-real-fourier) and R from global memory.
#include "common.cuh"
#include "kernels.h"

namespace cyfa {

namespace {

constexpr int G = 4;          // batch rows per block
constexpr int BATCH = 8;      // rows loaded per warp before they are used

template <int D, typename TI>
__global__ void __launch_bounds__(256) step_kernel(StepArgs a) {
    constexpr int VPL = D / 32;   // floats per lane per state row
    const int h = blockIdx.y, b0 = blockIdx.x * G;
    const int ng = min(G, a.B - b0);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    __shared__ float s_ct[MA], s_st[MA];
    __shared__ float s_q[G][D], s_k[G][D], s_v[G][D];
    __shared__ float s_a[G][MS], s_o1[G][MS], s_z[G][MS], s_u[G][MS], s_l[G][MS], s_y[G][MS];
    __shared__ float s_cs[G][64], s_sn[G][64];
    __shared__ float s_alpha[G], s_inv[G];
    __shared__ double s_lam[G];
    __shared__ float s_opart[2][G][D];

    const TI* Q = (const TI*)a.q;
    const TI* K = (const TI*)a.k;
    const TI* V = (const TI*)a.v;
    if (tid < MA) {
        float s, c;
        sincospif((float)tid * (2.f / 127.f), &s, &c);
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
    // clock, gates and rotation angles: thread (g, j) with j = 0 for the DC entry
    {
        const int g = tid >> 6, j = tid & 63;
        if (g < ng) {
            const size_t bh = (size_t)(b0 + g) * a.H + h;
            const double lam_new = a.lambda[bh] + (double)sigmoidf_(a.clock_logit[bh]);
            const float lam = (float)(lam_new - 127.0 * floor(lam_new / 127.0));
            const float beta = sigmoidf_(a.beta_logit[bh]);
            if (j == 0) {
                s_alpha[g] = expf(-a.A[h] * softplusf_(a.decay_logit[bh]));
                s_lam[g] = lam_new;
                s_a[g][0] = beta * INV_SQRT_M;
                s_a[g][127] = 0.f;
                s_cs[g][0] = 1.f;
                s_sn[g][0] = 0.f;
            } else {
                float s, c;
                sincospif(phase_pi(lam, j), &s, &c);
                s_cs[g][j] = c;
                s_sn[g][j] = s;
                s_a[g][2 * j - 1] = beta * SQRT_2_OVER_M * c;
                s_a[g][2 * j] = -beta * SQRT_2_OVER_M * s;
            }
        }
    }
    __syncthreads();

    // Kbar <- alpha Kbar + a k^T ; o' = Kbar (s q).  Warps 2g and 2g+1 own batch row g; warp
    // (2g + half) owns state rows r = half + 2 i.
    const int wg = warp >> 1, half = warp & 1;
    if (wg < ng) {
        const int g = wg;
        float* Kb = a.Kbar + ((size_t)(b0 + g) * a.H + h) * MS * D;
        const float alpha = s_alpha[g];
        float qv[VPL], kv[VPL];
#pragma unroll
        for (int u = 0; u < VPL; ++u) {
            qv[u] = s_q[g][lane * VPL + u];
            kv[u] = s_k[g][lane * VPL + u];
        }
        for (int i0 = 0; i0 < MS / 2; i0 += BATCH) {
            float x[BATCH][VPL];
#pragma unroll
            for (int bb = 0; bb < BATCH; ++bb) {
                const int r = half + 2 * (i0 + bb);
                if constexpr (VPL == 4) {
                    const float4 t = *reinterpret_cast<const float4*>(Kb + r * D + lane * 4);
                    x[bb][0] = t.x; x[bb][1] = t.y; x[bb][2] = t.z; x[bb][3] = t.w;
                } else {
                    const float2 t = *reinterpret_cast<const float2*>(Kb + r * D + lane * 2);
                    x[bb][0] = t.x; x[bb][1] = t.y;
                }
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
                if constexpr (VPL == 4) {
                    *reinterpret_cast<float4*>(Kb + r * D + lane * 4) =
                        make_float4(x[bb][0], x[bb][1], x[bb][2], x[bb][3]);
                } else {
                    *reinterpret_cast<float2*>(Kb + r * D + lane * 2) = make_float2(x[bb][0], x[bb][1]);
                }
                dot = warp_sum(dot);
                if (lane == 0) s_o1[g][r] = dot;
            }
        }
    }
    __syncthreads();

    // middle readout (Sec. 3.3 Eq. cyfa-two-pass, middle line) for the G rows:
    // z = U(lam) o'; u = Phi z; l = R u; p = softmax(l); y' = R^T p; y = Phi^T y'; o'' = U(-lam) y
    {
        const int g = tid >> 6, j = tid & 63;
        if (g < ng) {
            if (j == 0) {
                s_z[g][0] = s_o1[g][0];
                s_z[g][127] = 0.f;
            } else {
                const float c = s_cs[g][j], sn = s_sn[g][j];
                const float xc = s_o1[g][2 * j - 1], xs = s_o1[g][2 * j];
                s_z[g][2 * j - 1] = c * xc - sn * xs;
                s_z[g][2 * j] = sn * xc + c * xs;
            }
        }
    }
    __syncthreads();
    for (int e = tid; e < G * MS; e += 256) {   // u_r = z_0/sqrt(m) + sqrt(2/m) sum_j (...)
        const int g = e >> 7, r = e & 127;
        if (g < ng && r < MA) {
            float acc = 0.f;
            int idx = 0;
            for (int j = 1; j <= NPAIR; ++j) {
                idx += r;
                if (idx >= MA) idx -= MA;
                acc = fmaf(s_z[g][2 * j - 1], s_ct[idx], acc);
                acc = fmaf(s_z[g][2 * j], s_st[idx], acc);
            }
            s_u[g][r] = s_z[g][0] * INV_SQRT_M + SQRT_2_OVER_M * acc;
        }
    }
    __syncthreads();
    const float* Rh = a.R + (size_t)h * MA * MA;
    for (int i = warp; i < MA; i += 8) {   // l_i = sum_r R[i][r] u_r, one R row per warp
        float rv[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int r = lane + 32 * k;
            rv[k] = r < MA ? Rh[i * MA + r] : 0.f;
        }
        for (int g = 0; g < ng; ++g) {
            float acc = 0.f;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int r = lane + 32 * k;
                if (r < MA) acc = fmaf(rv[k], s_u[g][r], acc);
            }
            acc = warp_sum(acc);
            if (lane == 0) s_l[g][i] = acc;
        }
    }
    __syncthreads();
    if (warp < ng) {
        const int g = warp;
        float mx = -INFINITY;
        for (int i = lane; i < MA; i += 32) mx = fmaxf(mx, s_l[g][i]);
        mx = warp_max(mx);
        float sum = 0.f;
        for (int i = lane; i < MA; i += 32) {
            const float e = expf(s_l[g][i] - mx);
            s_l[g][i] = e;
            sum += e;
        }
        sum = warp_sum(sum);
        if (lane == 0) s_inv[g] = 1.f / sum;
    }
    __syncthreads();
    {   // y'_r = sum_i R[i][r] p_i, thread (r, half): rows g = half, half + 2
        const int r = tid & 127, half = tid >> 7;
        if (r < MA) {
            float acc0 = 0.f, acc1 = 0.f;
            const int g0 = half, g1 = half + 2;
            for (int i = 0; i < MA; ++i) {
                const float rv = Rh[i * MA + r];
                acc0 = fmaf(rv, s_l[g0][i], acc0);
                acc1 = fmaf(rv, s_l[g1][i], acc1);
            }
            if (g0 < ng) s_u[g0][r] = acc0 * s_inv[g0];
            if (g1 < ng) s_u[g1][r] = acc1 * s_inv[g1];
        }
    }
    __syncthreads();
    {   // y = Phi^T y', then o'' = U(-lam) y on the pair (2j-1, 2j)
        const int g = tid >> 6, j = tid & 63;
        if (g < ng) {
            if (j == 0) {
                float ac = 0.f;
                for (int r = 0; r < MA; ++r) ac += s_u[g][r];
                s_y[g][0] = ac * INV_SQRT_M;
                s_y[g][127] = 0.f;
            } else {
                float ac = 0.f, as = 0.f;
                int idx = 0;
                for (int r = 0; r < MA; ++r) {
                    ac = fmaf(s_u[g][r], s_ct[idx], ac);
                    as = fmaf(s_u[g][r], s_st[idx], as);
                    idx += j;
                    if (idx >= MA) idx -= MA;
                }
                const float yc = SQRT_2_OVER_M * ac, ys = SQRT_2_OVER_M * as;
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
        float* Vb = a.Vbar + ((size_t)(b0 + g) * a.H + h) * MS * D;
        const float alpha = s_alpha[g];
        float vv[VPL], oacc[VPL];
#pragma unroll
        for (int u = 0; u < VPL; ++u) {
            vv[u] = s_v[g][lane * VPL + u];
            oacc[u] = 0.f;
        }
        for (int i0 = 0; i0 < MS / 2; i0 += BATCH) {
            float x[BATCH][VPL];
#pragma unroll
            for (int bb = 0; bb < BATCH; ++bb) {
                const int r = half + 2 * (i0 + bb);
                if constexpr (VPL == 4) {
                    const float4 t = *reinterpret_cast<const float4*>(Vb + r * D + lane * 4);
                    x[bb][0] = t.x; x[bb][1] = t.y; x[bb][2] = t.z; x[bb][3] = t.w;
                } else {
                    const float2 t = *reinterpret_cast<const float2*>(Vb + r * D + lane * 2);
                    x[bb][0] = t.x; x[bb][1] = t.y;
                }
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
                if constexpr (VPL == 4) {
                    *reinterpret_cast<float4*>(Vb + r * D + lane * 4) =
                        make_float4(x[bb][0], x[bb][1], x[bb][2], x[bb][3]);
                } else {
                    *reinterpret_cast<float2*>(Vb + r * D + lane * 2) = make_float2(x[bb][0], x[bb][1]);
                }
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

}  // namespace

cudaError_t launch_step(const StepArgs& a, cudaStream_t st) {
    const dim3 grid((a.B + G - 1) / G, a.H);
    if (a.D == 128) {
        if (a.bf16) { LaunchScope ls_("decode_step", st); step_kernel<128, __nv_bfloat16><<<grid, 256, 0, st>>>(a); }
        else { LaunchScope ls_("decode_step", st); step_kernel<128, float><<<grid, 256, 0, st>>>(a); }
    } else if (a.D == 64) {
        if (a.bf16) { LaunchScope ls_("decode_step", st); step_kernel<64, __nv_bfloat16><<<grid, 256, 0, st>>>(a); }
        else { LaunchScope ls_("decode_step", st); step_kernel<64, float><<<grid, 256, 0, st>>>(a); }
    } else {
        return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace cyfa
