// Variants of cyfa_prepare: variable-length (packed) sequences and the fixed-rate clock.
//
// Fixed rate (App. A, Fixed-Rate Specialization, Eq. app-constant-rate-profile): the clock
// increment is the constant delta = 1/rho, so lambda_t = lambda0 + t / rho in closed form and no
// prefix sum over the clock logits is needed.
//
// Packed sequences: one stream of T tokens [1, T, H] holding nseq sequences back to back, sequence
// j on tokens [cu[j], cu[j+1]).  Every sequence starts from its own clock origin lambda0[j] and
// from the zero state.  The clock restarts by a segmented prefix sum (fp64).  The state restarts
// through the decay alone: at every sequence start r > 0 the chunk-local cumulative log-decay
// g_cum drops by RESET (64 nats) for the rest of r's chunk, so every decay factor exp(g_t - g_s)
// of the chunk form (App. B, Eq. app-chunk-decay) that spans r carries exp(-64) = 1.6e-28, and
// no contribution of an earlier sequence (through the intra-chunk products, the chunk-start
// state or the chunk-end state) survives in fp32.  g_cum stays non-increasing, so every decay
// factor the chunk kernels form remains <= 1.  Within a sequence the factors are unchanged up to
// one extra fp32 rounding of g at magnitude 64 n (n the number of starts in the chunk so far).
// The gradients need no change: every pair of tokens that spans a sequence start carries the
// vanishing factor, so the reverse cumulative sums of the decay and clock gradients (App. D.1
// Eq. app-clock-gradient-accumulation) pick up only cancelling terms from later sequences.
#include "../../include/cyfa.h"
#include "common.cuh"
#include "kernels.h"

namespace cyfa {

namespace {

constexpr float RESET = 64.f;   // nats of log-decay added at a sequence start (exp(-64) ~ 1.6e-28)

static __device__ int g_prep_err;

// First j in [0, n] with cu[j] >= x (cu has n + 1 entries); bounded by log2(n + 1) + 1 steps.
__device__ __forceinline__ int lower_bound_i(const int* cu, int n, int x) {
    int lo = 0, hi = n + 1;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (cu[mid] < x) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}
// Index of the sequence holding token t: the last j < n with cu[j] <= t (clamped to [0, n-1]).
__device__ __forceinline__ int seq_of(const int* cu, int n, int t) {
    int lo = 0, hi = n + 1;   // first j with cu[j] > t
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (cu[mid] <= t) lo = mid + 1;
        else hi = mid;
    }
    return min(max(lo - 1, 0), n - 1);
}

// Segmented sum: (flag, sum) of a token range is (a sequence starts in it, the sum from its last
// start to its end, or the whole sum when none starts in it).
struct Seg {
    int f;
    double s;
};
__device__ __forceinline__ Seg seg_join(Seg a, Seg b) { return {a.f | b.f, b.f ? b.s : a.s + b.s}; }

struct VarArgs {
    PrepareArgs p;     // p.s.B == 1 for packed sequences
    const int* cu;     // [nseq + 1] (device), nullptr for the dense fixed-rate variant
    int nseq;
    double rho;        // fixed rate: delta = 1 / rho when p.clock_logit == nullptr
    double* seg;       // [H][nseg][2] segment (flag, sum)
};

__device__ __forceinline__ double delta_of(const VarArgs& a, size_t gi) {
    return a.p.clock_logit ? (double)sigmoidf_(a.p.clock_logit[gi]) : 1.0 / a.rho;
}

// Marks the sequence starts of the block's tokens [t0, t0 + len) in s_seq (sequence index, or -1).
__device__ void mark_starts(const VarArgs& a, int t0, int len, int* s_seq) {
    for (int i = threadIdx.x; i < len; i += blockDim.x) s_seq[i] = -1;
    __syncthreads();
    const int n = a.nseq;
    const int j0 = lower_bound_i(a.cu, n, t0), j1 = min(lower_bound_i(a.cu, n, t0 + len), n);
    for (int j = j0 + (int)threadIdx.x; j < j1; j += blockDim.x) {
        const int r = a.cu[j];
        if (r < a.cu[j + 1] && r >= t0 && r < t0 + len) s_seq[r - t0] = j;   // non-empty only
    }
    __syncthreads();
}

// The value a token adds to the segmented clock sum: delta, plus the sequence's clock origin at
// its start.
__device__ __forceinline__ double clock_term(const VarArgs& a, int h, int seq, double d) {
    return d + ((seq >= 0 && a.p.lambda0) ? a.p.lambda0[(size_t)seq * a.p.s.H + h] : 0.0);
}

__global__ void __launch_bounds__(256) prepv_partial_kernel(VarArgs a, int nseg) {
    const int seg = blockIdx.x, h = blockIdx.y;
    const int H = a.p.s.H, T = a.p.s.T;
    const int t0 = seg * PREP_SEG, len = min(PREP_SEG, T - t0);
    __shared__ int s_seq[PREP_SEG];
    __shared__ Seg s_w[8];
    if (seg == 0 && h == 0) {   // the offsets must be a non-decreasing cover of [0, T)
        const int n = a.nseq;
        for (int j = threadIdx.x; j < n; j += blockDim.x)
            if (a.cu[j] > a.cu[j + 1]) atomicExch(&g_prep_err, CYFA_ERR_ARG);
        if (threadIdx.x == 0 && (a.cu[0] != 0 || a.cu[n] != T)) atomicExch(&g_prep_err, CYFA_ERR_ARG);
    }
    mark_starts(a, t0, len, s_seq);
    Seg acc = {0, 0.0};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int i = 4 * threadIdx.x + u;
        if (i < len) {
            const int sq = s_seq[i];
            const double x = clock_term(a, h, sq, delta_of(a, (size_t)(t0 + i) * H + h));
            acc = seg_join(acc, Seg{sq >= 0, x});
        }
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {   // ordered reduction: lanes below come first
        Seg y;
        y.f = __shfl_up_sync(0xffffffffu, acc.f, o);
        y.s = __shfl_up_sync(0xffffffffu, acc.s, o);
        if (lane >= o) acc = seg_join(y, acc);
    }
    if (lane == 31) s_w[warp] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        Seg t = s_w[0];
        for (int w = 1; w < 8; ++w) t = seg_join(t, s_w[w]);
        a.seg[((size_t)h * nseg + seg) * 2] = t.f;
        a.seg[((size_t)h * nseg + seg) * 2 + 1] = t.s;
    }
}

// Clock (segmented fp64 scan, reduced mod m), chunk-local log-decay with the reset offsets, and
// write strengths.  VARLEN = false: the dense fixed-rate clock lambda0[b,h] + t / rho.
template <bool VARLEN>
__global__ void __launch_bounds__(256) prepv_scan_kernel(VarArgs a, int nseg) {
    const int seg = blockIdx.x, bh = blockIdx.y;
    const int H = a.p.s.H, T = a.p.s.T, C = a.p.s.C;
    const int b = bh / H, h = bh % H;
    const int t0 = seg * PREP_SEG, len = min(PREP_SEG, T - t0);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __shared__ int s_seq[VARLEN ? PREP_SEG : 1];
    __shared__ Seg s_w[8];
    __shared__ Seg s_carry;
    const float Ah = a.p.A[h];

    double lamv[4];
    int nres[4];
    float lp[4];
    float lpref = 0.f;
    int cres = 0;
    if (VARLEN) {
        mark_starts(a, t0, len, s_seq);
        if (warp == 0) {   // carry: the segmented sum of every earlier segment, in order
            const int per = (seg + 31) / 32;
            Seg x = {0, 0.0};
            for (int k = lane * per; k < min(seg, (lane + 1) * per); ++k) {
                const double* p = a.seg + ((size_t)h * nseg + k) * 2;
                x = seg_join(x, Seg{(int)p[0], p[1]});
            }
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                Seg y;
                y.f = __shfl_up_sync(0xffffffffu, x.f, o);
                y.s = __shfl_up_sync(0xffffffffu, x.s, o);
                if (lane >= o) x = seg_join(y, x);
            }
            if (lane == 31) s_carry = x;
        }
        if (seg == 0)   // empty sequences: their end clock is their origin
            for (int j = threadIdx.x; j < a.nseq; j += blockDim.x)
                if (a.cu[j] == a.cu[j + 1] && a.p.lambda_end)
                    a.p.lambda_end[(size_t)j * H + h] = a.p.lambda0 ? a.p.lambda0[(size_t)j * H + h] : 0.0;
        // thread-local segmented scan of the clock over its four tokens
        Seg acc = {0, 0.0};
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = 4 * threadIdx.x + u;
            int sq = -1;
            double x = 0.0;
            float la = 0.f;
            if (i < len) {
                const size_t gi = (size_t)(t0 + i) * H + h;
                sq = s_seq[i];
                x = clock_term(a, h, sq, delta_of(a, gi));
                la = -Ah * softplusf_(a.p.decay_logit[gi]);
                a.p.beta[gi] = sigmoidf_(a.p.beta_logit[gi]);
            }
            acc = seg_join(acc, Seg{sq >= 0, x});
            lamv[u] = acc.s;
            nres[u] = (sq >= 0 && t0 + i > 0) ? 1 : 0;
            lpref += la;
            lp[u] = lpref;
        }
        // block-wide exclusive segmented scan of the per-thread totals, after the carry
        Seg incl = acc;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            Seg y;
            y.f = __shfl_up_sync(0xffffffffu, incl.f, o);
            y.s = __shfl_up_sync(0xffffffffu, incl.s, o);
            if (lane >= o) incl = seg_join(y, incl);
        }
        if (lane == 31) s_w[warp] = incl;
        __syncthreads();
        Seg ex = s_carry;
        for (int w = 0; w < warp; ++w) ex = seg_join(ex, s_w[w]);
        Seg pl;
        pl.f = __shfl_up_sync(0xffffffffu, incl.f, 1);
        pl.s = __shfl_up_sync(0xffffffffu, incl.s, 1);
        if (lane > 0) ex = seg_join(ex, pl);
        // token u: value from the last start at or before it within the thread, else carry + own
        bool seen = false;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = 4 * threadIdx.x + u;
            seen = seen || (i < len && s_seq[i] >= 0);
            if (!seen) lamv[u] += ex.s;
        }
        cres = nres[0] + nres[1] + nres[2] + nres[3];
    } else {
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = 4 * threadIdx.x + u;
            float la = 0.f;
            if (i < len) {
                const size_t gi = ((size_t)b * T + t0 + i) * H + h;
                la = -Ah * softplusf_(a.p.decay_logit[gi]);
                a.p.beta[gi] = sigmoidf_(a.p.beta_logit[gi]);
            }
            lamv[u] = (a.p.lambda0 ? a.p.lambda0[bh] : 0.0) + (double)(t0 + i + 1) / a.rho;
            nres[u] = 0;
            lpref += la;
            lp[u] = lpref;
        }
    }
    // chunk-local scans (a chunk spans C/4 consecutive lanes of one warp): log-decay and the
    // number of sequence starts
    const int seg_lanes = C / 4;
    float tot = lp[3];
    int rtot = cres;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, tot, o);
        const int yr = __shfl_up_sync(0xffffffffu, rtot, o);
        if (o < seg_lanes && (lane % seg_lanes) >= o) {
            tot += y;
            rtot += yr;
        }
    }
    const float gex = tot - lp[3];
    int rex = rtot - cres;
    int cur_seq = VARLEN ? seq_of(a.cu, a.nseq, t0 + 4 * (int)threadIdx.x) : 0;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int i = 4 * threadIdx.x + u;
        rex += nres[u];
        if (i < len) {
            const size_t gi = ((size_t)b * T + t0 + i) * H + h;
            const double fm = (double)a.p.s.sl.m;
            double lm = lamv[u];
            lm = fma(-fm, floor(lm * (1.0 / fm)), lm);
            if (lm < 0.0) lm += fm;
            else if (lm >= fm) lm -= fm;
            a.p.lam_mod[gi] = (float)lm;
            a.p.g_cum[gi] = (gex + lp[u]) - RESET * (float)rex;
            if (VARLEN) {
                if (s_seq[i] >= 0) cur_seq = s_seq[i];
                const int t = t0 + i;
                if (a.p.lambda_end && a.cu[cur_seq + 1] == t + 1)
                    a.p.lambda_end[(size_t)cur_seq * H + h] = lamv[u];
            } else if (a.p.lambda_end && t0 + i == T - 1) {
                a.p.lambda_end[bh] = lamv[u];
            }
        }
    }
}

}  // namespace

size_t prepare_varlen_workspace(const Shape& s) {
    const size_t nseg = (s.T + PREP_SEG - 1) / PREP_SEG;
    return 2 * nseg * (size_t)s.H * sizeof(double);
}

cudaError_t launch_prepare_varlen(const PrepareArgs& p, const int* cu, int nseq, double rho,
                                  double* seg, cudaStream_t st) {
    VarArgs a;
    a.p = p;
    a.cu = cu;
    a.nseq = nseq;
    a.rho = rho;
    a.seg = seg;
    const int nseg = (p.s.T + PREP_SEG - 1) / PREP_SEG;
    dim3 grid(nseg, p.s.H);
    { LaunchScope ls_("prepv_partial", st); prepv_partial_kernel<<<grid, 256, 0, st>>>(a, nseg); }
    { LaunchScope ls_("prepv_scan", st); prepv_scan_kernel<true><<<grid, 256, 0, st>>>(a, nseg); }
    return cudaGetLastError();
}

cudaError_t launch_prepare_fixed_rate(const PrepareArgs& p, double rho, cudaStream_t st) {
    VarArgs a;
    a.p = p;
    a.cu = nullptr;
    a.nseq = 0;
    a.rho = rho;
    a.seg = nullptr;
    const int nseg = (p.s.T + PREP_SEG - 1) / PREP_SEG;
    dim3 grid(nseg, p.s.B * p.s.H);
    { LaunchScope ls_("prepf_scan", st); prepv_scan_kernel<false><<<grid, 256, 0, st>>>(a, nseg); }
    return cudaGetLastError();
}

cudaError_t prep_read_error(cudaStream_t st, int* err) {
    cudaError_t e = cudaMemcpyFromSymbolAsync(err, g_prep_err, sizeof(int), 0,
                                              cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return e;
    e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return e;
    if (*err) {
        const int zero = 0;
        e = cudaMemcpyToSymbol(g_prep_err, &zero, sizeof(int));
    }
    return e;
}

}  // namespace cyfa
