// cyfa_prepare kernels: clock prefix sum (fp64 carry) reduced mod m, chunk-local cumulative
// log-decays, and write strengths.  Sec. 3.1 Eq. cyfa-cumulative-clock; Sec. 3.4 forget gate;
// App. B Eq. app-chunk-decay (gamma^r as exp of a chunk-local cumulative sum of log alpha).
//
// Layout: gates are [B, T, H] fp32.  Two launches: per (b, h, 1024-token segment) fp64 sums of
// delta, then a block scan per segment that adds the sums of the segments before it.
#include <mutex>

#include "../../include/cyfa.h"
#include "common.cuh"
#include "kernels.h"

namespace cyfa {

namespace {

__device__ __forceinline__ double warp_sum_d(double x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__global__ void __launch_bounds__(256) prep_partial_kernel(PrepareArgs a, int nseg) {
    const int seg = blockIdx.x, bh = blockIdx.y;
    const int H = a.s.H, T = a.s.T;
    const int b = bh / H, h = bh % H;
    const int t0 = seg * PREP_SEG;
    const int len = min(PREP_SEG, T - t0);
    double acc = 0.0;
    for (int i = threadIdx.x; i < len; i += blockDim.x)
        acc += (double)sigmoidf_(a.clock_logit[((size_t)b * T + t0 + i) * H + h]);
    __shared__ double red[8];
    acc = warp_sum_d(acc);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < 8; ++w) t += red[w];
        a.seg_sum[(size_t)bh * nseg + seg] = t;
    }
}

__global__ void __launch_bounds__(256) prep_scan_kernel(PrepareArgs a, int nseg) {
    const int seg = blockIdx.x, bh = blockIdx.y;
    const int H = a.s.H, T = a.s.T, C = a.s.C;
    const int b = bh / H, h = bh % H;
    const int t0 = seg * PREP_SEG;
    const int len = min(PREP_SEG, T - t0);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __shared__ double s_base;
    __shared__ double s_wtot[8];

    if (warp == 0) {
        double x = 0.0;
        for (int s = lane; s < seg; s += 32) x += a.seg_sum[(size_t)bh * nseg + s];
        x = warp_sum_d(x);
        if (lane == 0) s_base = x + (a.lambda0 ? a.lambda0[bh] : 0.0);
    }

    const float Ah = a.A[h];
    double loc[4];
    float lp[4];
    double pref = 0.0;
    float lpref = 0.f;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int i = 4 * threadIdx.x + u;
        float d = 0.f, la = 0.f;
        if (i < len) {
            const size_t gi = ((size_t)b * T + t0 + i) * H + h;
            d = sigmoidf_(a.clock_logit[gi]);
            la = -Ah * softplusf_(a.decay_logit[gi]);
            a.beta[gi] = sigmoidf_(a.beta_logit[gi]);
        }
        pref += (double)d;
        loc[u] = pref;
        lpref += la;
        lp[u] = lpref;
    }
    // block-wide exclusive scan of the per-thread delta totals (fp64)
    double incl = pref;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const double y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) s_wtot[warp] = incl;
    // chunk-local scan of log alpha: a chunk spans C/4 consecutive lanes of one warp
    const int seg_lanes = C / 4;
    float tot = lp[3];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, tot, o);
        if (o < seg_lanes && (lane % seg_lanes) >= o) tot += y;
    }
    const float gex = tot - lp[3];
    __syncthreads();
    double wex = 0.0;
    for (int w = 0; w < warp; ++w) wex += s_wtot[w];
    const double excl = s_base + wex + (incl - pref);
    // clock mod m: the clock before this thread's first token is reduced once in fp64 (one
    // multiply by 1/m, no divide); its four tokens add their increments in fp64 (together < 4,
    // so at most one wrap) and are rounded to fp32 once
    const double fm = (double)a.s.sl.m, inv_m = 1.0 / fm;
    double bm = fma(-fm, floor(excl * inv_m), excl);
    if (bm < 0.0) bm += fm;
    else if (bm >= fm) bm -= fm;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int i = 4 * threadIdx.x + u;
        if (i < len) {
            const size_t gi = ((size_t)b * T + t0 + i) * H + h;
            double lm = bm + loc[u];
            if (lm >= fm) lm -= fm;
            a.lam_mod[gi] = (float)lm;
            a.g_cum[gi] = gex + lp[u];
            if (a.lambda_end && t0 + i == T - 1) a.lambda_end[bh] = excl + loc[u];
        }
    }
}

}  // namespace

size_t prepare_workspace(const Shape& s) {
    const size_t nseg = (s.T + PREP_SEG - 1) / PREP_SEG;
    return nseg * (size_t)s.B * s.H * sizeof(double);
}

cudaError_t launch_prepare(const PrepareArgs& a, cudaStream_t st) {
    const int nseg = (a.s.T + PREP_SEG - 1) / PREP_SEG;
    dim3 grid(nseg, a.s.B * a.s.H);
    { LaunchScope ls_("prep_partial", st); prep_partial_kernel<<<grid, 256, 0, st>>>(a, nseg); }
    { LaunchScope ls_("prep_scan", st); prep_scan_kernel<<<grid, 256, 0, st>>>(a, nseg); }
    return cudaGetLastError();
}

}  // namespace cyfa

// ---------------------------------------------------------------------------------------
// cyfa_prepare_noalloc: cyfa_prepare without a caller workspace.
//
// Some callers cannot give the library any device memory beyond the tensors themselves: an
// inference server or plugin host that reserves all device memory up front through its own
// allocator and forbids later cudaMalloc calls, or a latency-critical loop that must never
// allocate.  This entry point runs the same two prepare kernels, but the per-segment partial
// sums live in a fixed array compiled into the library instead of a workspace.
//
// The array is a file-scope __device__ variable: every GPU that loads the library holds it
// (256 KiB) until the process exits.  Its host-side name is only a stand-in, never a device
// address, so the address is looked up with cudaGetSymbolAddress once per device, with that
// device current, on the first call made on the device.
namespace cyfa {
namespace {

constexpr int kNoAllocMaxSegSums = 32768;   // B * H * ceil(T / 1024) fp64 partial sums
static __device__ __align__(256) double g_noalloc_seg_sum[kNoAllocMaxSegSums];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
double* g_noalloc_ptr[kMaxDevices] = {};

// Device address of g_noalloc_seg_sum on the current device (looked up once per device).
cudaError_t noalloc_scratch(double** out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_seg_sum);
        if (e != cudaSuccess) return e;
        g_noalloc_ptr[dev] = static_cast<double*>(p);
    }
    *out = g_noalloc_ptr[dev];
    return cudaSuccess;
}

}  // namespace
}  // namespace cyfa

extern "C" int cyfa_prepare_noalloc(const cyfa_dims_t* dims, const float* clock_logit,
                                    const float* decay_logit, const float* beta_logit,
                                    const float* A, const double* lambda0, float* lam_mod,
                                    float* g_cum, float* beta, double* lambda_end, void* stream) {
    using namespace cyfa;
    const int rc = check_dims(dims, true);   // the same argument checks as cyfa_prepare
    if (rc) return rc;
    if (!clock_logit || !decay_logit || !beta_logit || !A || !lam_mod || !g_cum || !beta)
        return CYFA_ERR_ARG;
    const long long nseg = (dims->T + PREP_SEG - 1) / PREP_SEG;
    if ((long long)dims->B * dims->H * nseg > kNoAllocMaxSegSums) return CYFA_ERR_WORKSPACE;
    double* scratch = nullptr;
    if (noalloc_scratch(&scratch) != cudaSuccess) return CYFA_ERR_CUDA;
    PrepareArgs a;
    a.s.B = dims->B;
    a.s.T = dims->T;
    a.s.H = dims->H;
    a.s.D = dims->dk;
    a.s.C = dims->chunk;
    a.s.Cg = dims->chunk;
    a.s.scale = dims->scale;
    a.s.bf16 = dims->dtype == CYFA_DTYPE_BF16;
    a.s.sl = make_slots(dims->m);
    a.clock_logit = clock_logit;
    a.decay_logit = decay_logit;
    a.beta_logit = beta_logit;
    a.A = A;
    a.lambda0 = lambda0;
    a.lam_mod = lam_mod;
    a.g_cum = g_cum;
    a.beta = beta;
    a.lambda_end = lambda_end;
    a.seg_sum = scratch;   // every entry is written by the first kernel before the second reads it
    return launch_prepare(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? CYFA_OK
                                                                                 : CYFA_ERR_CUDA;
}
