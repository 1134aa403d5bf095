// cyfa_step: one decode token against the persistent fp32 states (Sec. 3.2 Eq.
// cyfa-absolute-recurrence and Eq. cyfa-absolute-readout applied to a single token).
//
// One 256-thread block per (b, h).  The step is HBM-bound: each block streams its 64 KB Kbar
// and 64 KB Vbar (D = 128) once in and once out with 16-byte accesses.  The middle readout
// applies Phi through a 127-entry cosine / sine table (entry (j r) mod m of Eq.
// app-real-fourier) and R straight from global memory (shared by every batch row of a head,
// so it stays in L2).
#include "common.cuh"
#include "kernels.h"

namespace cyfa {

namespace {

template <int D, typename TI>
__global__ void __launch_bounds__(256) step_kernel(StepArgs a) {
    const int bh = blockIdx.x, h = bh % a.H;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    __shared__ float s_a[MS], s_q[D], s_k[D], s_v[D], s_o1[MS], s_z[MS], s_u[MS], s_l[MS],
        s_y[MS], s_ct[MA], s_st[MA];
    __shared__ float s_opart[8][D];
    __shared__ float s_cs[NPAIR + 1], s_sn[NPAIR + 1];
    __shared__ float s_alpha, s_red[2];

    const TI* Q = (const TI*)a.q;
    const TI* K = (const TI*)a.k;
    const TI* V = (const TI*)a.v;
    if (tid < D) {
        s_q[tid] = a.scale * ldf(Q, (size_t)bh * D + tid);
        s_k[tid] = ldf(K, (size_t)bh * D + tid);
        s_v[tid] = ldf(V, (size_t)bh * D + tid);
    }
    if (tid < MA) {
        float s, c;
        sincospif((float)tid * (2.f / 127.f), &s, &c);
        s_ct[tid] = c;
        s_st[tid] = s;
    }
    // clock, gates and rotation angles of this token
    double lam_new = 0.0;
    {
        const float delta = sigmoidf_(a.clock_logit[bh]);
        lam_new = a.lambda[bh] + (double)delta;
        const float lam = (float)(lam_new - 127.0 * floor(lam_new / 127.0));
        const float beta = sigmoidf_(a.beta_logit[bh]);
        if (tid == 0) s_alpha = expf(-a.A[h] * softplusf_(a.decay_logit[bh]));
        if (tid <= NPAIR) {
            float s = 0.f, c = 1.f;
            if (tid > 0) sincospif(phase_pi(lam, tid), &s, &c);
            s_cs[tid] = c;
            s_sn[tid] = s;
            if (tid == 0) {
                s_a[0] = beta * INV_SQRT_M;
                s_a[127] = 0.f;
            } else {
                s_a[2 * tid - 1] = beta * SQRT_2_OVER_M * c;
                s_a[2 * tid] = -beta * SQRT_2_OVER_M * s;
            }
        }
    }
    __syncthreads();
    const float alpha = s_alpha;

    // Kbar <- alpha Kbar + a k^T ; o' = Kbar (s q).  Warp w owns rows w, w+8, ...; lane owns
    // D/32 consecutive columns.
    constexpr int VPL = D / 32;  // floats per lane per row (4 for D = 128)
    float* Kb = a.Kbar + (size_t)bh * MS * D;
    float* Vb = a.Vbar + (size_t)bh * MS * D;
    float qv[VPL], kv[VPL];
#pragma unroll
    for (int u = 0; u < VPL; ++u) {
        qv[u] = s_q[lane * VPL + u];
        kv[u] = s_k[lane * VPL + u];
    }
#pragma unroll 4
    for (int r = warp; r < MS; r += 8) {
        float x[VPL];
        if constexpr (VPL == 4) {
            const float4 t = *reinterpret_cast<const float4*>(Kb + r * D + lane * 4);
            x[0] = t.x; x[1] = t.y; x[2] = t.z; x[3] = t.w;
        } else {
            const float2 t = *reinterpret_cast<const float2*>(Kb + r * D + lane * 2);
            x[0] = t.x; x[1] = t.y;
        }
        const float ar = s_a[r];
        float dot = 0.f;
#pragma unroll
        for (int u = 0; u < VPL; ++u) {
            x[u] = fmaf(alpha, x[u], ar * kv[u]);
            dot = fmaf(x[u], qv[u], dot);
        }
        if constexpr (VPL == 4) {
            *reinterpret_cast<float4*>(Kb + r * D + lane * 4) = make_float4(x[0], x[1], x[2], x[3]);
        } else {
            *reinterpret_cast<float2*>(Kb + r * D + lane * 2) = make_float2(x[0], x[1]);
        }
        dot = warp_sum(dot);
        if (lane == 0) s_o1[r] = dot;
    }
    __syncthreads();

    // middle readout: z = U(lam) o'; u = Phi z; l = R u; p = softmax(l); y' = R^T p;
    // y = Phi^T y'; o'' = U(-lam) y  (Sec. 3.3 Eq. cyfa-two-pass, middle line)
    if (tid <= NPAIR) {
        if (tid == 0) {
            s_z[0] = s_o1[0];
            s_z[127] = 0.f;
        } else {
            const float c = s_cs[tid], sn = s_sn[tid];
            const float xc = s_o1[2 * tid - 1], xs = s_o1[2 * tid];
            s_z[2 * tid - 1] = c * xc - sn * xs;
            s_z[2 * tid] = sn * xc + c * xs;
        }
    }
    __syncthreads();
    if (tid < MA) {  // u_r = z_0/sqrt(m) + sqrt(2/m) sum_j (z_{2j-1} cos + z_{2j} sin)(2 pi j r / m)
        float acc = 0.f;
        int idx = 0;
        for (int j = 1; j <= NPAIR; ++j) {
            idx += tid;
            if (idx >= MA) idx -= MA;
            acc = fmaf(s_z[2 * j - 1], s_ct[idx], acc);
            acc = fmaf(s_z[2 * j], s_st[idx], acc);
        }
        s_u[tid] = s_z[0] * INV_SQRT_M + SQRT_2_OVER_M * acc;
    }
    __syncthreads();
    const float* Rh = a.R + (size_t)h * MA * MA;
    for (int i = warp; i < MA; i += 8) {  // l_i = sum_r R[i][r] u_r
        float acc = 0.f;
        for (int r = lane; r < MA; r += 32) acc = fmaf(Rh[i * MA + r], s_u[r], acc);
        acc = warp_sum(acc);
        if (lane == 0) s_l[i] = acc;
    }
    __syncthreads();
    if (warp == 0) {
        float mx = -INFINITY;
        for (int i = lane; i < MA; i += 32) mx = fmaxf(mx, s_l[i]);
        mx = warp_max(mx);
        float sum = 0.f;
        for (int i = lane; i < MA; i += 32) {
            const float e = expf(s_l[i] - mx);
            s_l[i] = e;
            sum += e;
        }
        sum = warp_sum(sum);
        if (lane == 0) s_red[0] = 1.f / sum;
    }
    __syncthreads();
    if (tid < MA) {  // y'_r = sum_i R[i][r] p_i
        const float inv = s_red[0];
        float acc = 0.f;
        for (int i = 0; i < MA; ++i) acc = fmaf(Rh[i * MA + tid], s_l[i], acc);
        s_u[tid] = acc * inv;
    }
    __syncthreads();
    if (tid <= NPAIR) {  // y = Phi^T y'
        float ac = 0.f, as = 0.f;
        if (tid == 0) {
            for (int r = 0; r < MA; ++r) ac += s_u[r];
            s_y[0] = ac * INV_SQRT_M;
            s_y[127] = 0.f;
        } else {
            int idx = 0;
            for (int r = 0; r < MA; ++r) {
                ac = fmaf(s_u[r], s_ct[idx], ac);
                as = fmaf(s_u[r], s_st[idx], as);
                idx += tid;
                if (idx >= MA) idx -= MA;
            }
            // o'' = U(-lam) y on the pair (2j-1, 2j)
            const float yc = SQRT_2_OVER_M * ac, ys = SQRT_2_OVER_M * as;
            const float c = s_cs[tid], sn = s_sn[tid];
            s_y[2 * tid - 1] = c * yc + sn * ys;
            s_y[2 * tid] = -sn * yc + c * ys;
        }
    }
    __syncthreads();

    // Vbar <- alpha Vbar + a v^T ; o = Vbar^T o''
    float vv[VPL], oacc[VPL];
#pragma unroll
    for (int u = 0; u < VPL; ++u) {
        vv[u] = s_v[lane * VPL + u];
        oacc[u] = 0.f;
    }
#pragma unroll 4
    for (int r = warp; r < MS; r += 8) {
        float x[VPL];
        if constexpr (VPL == 4) {
            const float4 t = *reinterpret_cast<const float4*>(Vb + r * D + lane * 4);
            x[0] = t.x; x[1] = t.y; x[2] = t.z; x[3] = t.w;
        } else {
            const float2 t = *reinterpret_cast<const float2*>(Vb + r * D + lane * 2);
            x[0] = t.x; x[1] = t.y;
        }
        const float ar = s_a[r], yr = s_y[r];
#pragma unroll
        for (int u = 0; u < VPL; ++u) {
            x[u] = fmaf(alpha, x[u], ar * vv[u]);
            oacc[u] = fmaf(x[u], yr, oacc[u]);
        }
        if constexpr (VPL == 4) {
            *reinterpret_cast<float4*>(Vb + r * D + lane * 4) = make_float4(x[0], x[1], x[2], x[3]);
        } else {
            *reinterpret_cast<float2*>(Vb + r * D + lane * 2) = make_float2(x[0], x[1]);
        }
    }
#pragma unroll
    for (int u = 0; u < VPL; ++u) s_opart[warp][lane * VPL + u] = oacc[u];
    __syncthreads();
    if (tid < D) {
        float acc = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) acc += s_opart[w][tid];
        stf((TI*)a.o, (size_t)bh * D + tid, acc);
    }
    if (tid == 0) a.lambda[bh] = lam_new;
}

}  // namespace

cudaError_t launch_step(const StepArgs& a, cudaStream_t st) {
    const int grid = a.B * a.H;
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
