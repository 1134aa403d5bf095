/*
 * cyfa.h -- C ABI of the CyFA (Cyclic Flow Attention) core operator for GB300 (sm_103a).
 *
 * The operator is the absolute-clock form of CyFA (Sec. 3.2, Eq. cyfa-absolute-recurrence
 * and Eq. cyfa-absolute-readout), evaluated chunk-wise as two scalar-decay linear-attention
 * passes joined by a token-wise softmax readout (Sec. 3.3 Eq. cyfa-two-pass; App. B Eqs.
 * app-cyfa-key-chunk and app-cyfa-value-chunk).  Per (batch b, head h) and token t:
 *
 *   delta_t  = sigmoid(clock_logit_t)                     clock increment, Eq. clock_gradient_stabilization
 *   lambda_t = lambda_{t-1} + delta_t                     cumulative clock, Eq. cyfa-cumulative-clock
 *   alpha_t  = exp(-A_h softplus(decay_logit_t))          scalar forget gate, Sec. 3.4
 *   beta_t   = sigmoid(beta_logit_t)                      write strength (activation: this library's reading)
 *   a_t      = beta_t U(-lambda_t) b                      temporal write vector, Sec. 3.2
 *   Kbar_t   = alpha_t Kbar_{t-1} + a_t k_t^T             key state   [m x dk]
 *   Vbar_t   = alpha_t Vbar_{t-1} + a_t v_t^T             value state [m x dv]
 *   o'_t     = Kbar_t (scale q_t)
 *   o''_t    = U(-lambda_t) Phi^T R^T softmax(R Phi U(lambda_t) o'_t)
 *   o_t      = Vbar_t^T o''_t
 *
 * Threads: any host thread may call; the calls use the runtime's current device of the calling
 * thread (cudaSetDevice) and the caller's stream.
 *
 * Storage conventions (all row-major, caller-owned; the library never allocates):
 *   q, k, dq, dk      [B, T, H, dk]   bf16 or fp32 (dims.dtype)
 *   v, o, dO, dv      [B, T, H, dv]   bf16 or fp32
 *   *_logit, lam_mod, g_cum, beta, d_*_logit   [B, T, H] fp32
 *   A                 [H] fp32 (> 0)
 *   R, dR             [H, m, m] fp32
 *   Kbar, Vbar        [B, H, ms, dk] / [B, H, ms, dv] fp32 with ms = 128 storage rows for
 *                     m <= 127 and 256 above; rows in the order of the real Fourier basis of
 *                     App. A.1 Eq. app-real-fourier (DC, cos_1, sin_1, ..., cos_p, sin_p with
 *                     p = (m-1)/2) followed by ms - m padding rows that stay zero (App. A.7;
 *                     one row at m = 127 and at m = 255).
 *   lambda            [B, H] fp64 (the running clock)
 *   stream            a cudaStream_t passed as void*; every call is asynchronous on it.
 *
 * Shapes supported: odd m in 1..255 (128 storage rows up to m = 127, 256 above), dk = dv in
 * {64, 128, 256}, chunk in {64, 128}, T a positive multiple of chunk (for cyfa_prepare /
 * cyfa_chunk_fwd / cyfa_chunk_bwd), B * H <= 65535.  The tensor-core kernels take bf16 with
 * d = 128, 63 <= m <= 127 and T a multiple of 128; every other supported shape runs on the fp32
 * CUDA-core kernels.
 *
 * Errors: every entry point returns CYFA_OK (0) or a negative code.  Argument errors are
 * found on the host before anything is launched.  CYFA_ERR_TIMEOUT (a bounded wait expired)
 * and CYFA_ERR_RANGE (a non-finite value reached a result) are raised on the device and read
 * back by cyfa_check().
 */
#ifndef CYFA_H
#define CYFA_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
    CYFA_OK = 0,
    CYFA_ERR_ARG = -1,        /* null required pointer or non-positive size */
    CYFA_ERR_SHAPE = -2,      /* unsupported m, d, chunk, or T not a multiple of chunk */
    CYFA_ERR_ALIGN = -3,      /* a tensor pointer is not 16-byte aligned */
    CYFA_ERR_WORKSPACE = -4,  /* workspace null or smaller than cyfa_workspace_size() */
    CYFA_ERR_CUDA = -5,       /* a CUDA runtime call or launch failed */
    CYFA_ERR_TIMEOUT = -6,    /* a bounded device-side wait expired (see cyfa_check) */
    CYFA_ERR_UNSUPPORTED = -7,/* a valid request this build does not implement (no current
                                 call returns it; kept so codes stay stable) */
    CYFA_ERR_RANGE = -8       /* a non-finite value reached a result (see cyfa_check) */
};

enum { CYFA_DTYPE_BF16 = 0, CYFA_DTYPE_FP32 = 1 };

/* Which call a workspace is sized for. */
enum { CYFA_WS_PREPARE = 0, CYFA_WS_FWD = 1, CYFA_WS_BWD = 2, CYFA_WS_PREPARE_VARLEN = 3,
       CYFA_WS_MIXER = 4 };

typedef struct cyfa_dims {
    int B, T, H;   /* batch, sequence length, heads */
    int dk, dv;    /* head dims (dk == dv) */
    int m;         /* active relative-time slots: odd, 1..255 (the paper's default is 127) */
    int chunk;     /* tokens per chunk: 64 or 128 */
    float scale;   /* dot-product scale s; the query enters the key pass as s*q */
    int dtype;     /* CYFA_DTYPE_BF16 or CYFA_DTYPE_FP32 for q, k, v, o, dO, dq, dk, dv */
    int flags;     /* CYFA_FLAG_* bits; 0 for the default kernels */
} cyfa_dims_t;

/* dims.flags: run the chunk calls on the fp32 CUDA-core kernels even where the tensor-core
 * kernels apply (bf16, d = 128, 63 <= m <= 127, T a multiple of 128).  Slower; exact fp32
 * intermediates. */
enum { CYFA_FLAG_CUDA_CORES = 1 };

/* Library version as 10000*major + 100*minor + patch. */
int cyfa_version(void);

/* Human-readable text for an error code (static storage, never NULL). */
const char* cyfa_error_string(int code);

/* Bytes of device workspace the call `which` (CYFA_WS_*) needs for these dims. */
int cyfa_workspace_size(const cyfa_dims_t* dims, int which, size_t* bytes);

/*
 * cyfa_prepare -- per-token gates and the absolute-clock coordinates (Sec. 3.1 Eq.
 * cyfa-cumulative-clock, Sec. 3.4, App. B chunk-local log-decays of Eq. app-chunk-decay).
 *
 *   lam_mod[b,t,h] = lambda_t mod m, with lambda_t = lambda0[b,h] + sum_{u<=t} delta_u
 *                    carried in fp64; U is m-periodic (Prop. 1) so the reduction is exact.
 *   g_cum[b,t,h]   = sum of log alpha_u over the tokens u <= t of t's chunk (<= 0).
 *   beta[b,t,h]    = sigmoid(beta_logit).
 *   lambda_end[b,h] (nullable) = lambda_T in fp64, the clock a following cyfa_step continues.
 * lambda0 may be NULL (clock origin 0; Prop. 6 makes the origin arbitrary).
 * Needs cyfa_workspace_size(CYFA_WS_PREPARE) bytes of workspace.
 */
int cyfa_prepare(const cyfa_dims_t* dims, const float* clock_logit, const float* decay_logit,
                 const float* beta_logit, const float* A, const double* lambda0,
                 float* lam_mod, float* g_cum, float* beta, double* lambda_end,
                 void* workspace, size_t workspace_bytes, void* stream);

/*
 * cyfa_prepare_fixed_rate -- cyfa_prepare for the fixed-rate clock delta_t = 1 / rho (App. A,
 * Fixed-Rate Specialization and Relation to BLA, Eq. app-constant-rate-profile: with a constant
 * increment the relative-time profile is the Fourier-Dirichlet profile of Blurry Window
 * Attention).  lambda_t = lambda0[b,h] + t / rho (t = 1..T) in fp64 closed form, reduced mod m:
 * there are no clock logits and no prefix sum, so no workspace.  g_cum, beta and lambda_end as in
 * cyfa_prepare.  rho > 0 (CYFA_ERR_ARG otherwise).  The chunk calls take the results unchanged;
 * cyfa_chunk_bwd then gets clock_logit = d_clock_logit = NULL.  A decode step of the same model
 * is cyfa_step with clock logit -ln(rho - 1) (+inf for rho = 1), whose sigmoid is 1 / rho.
 */
int cyfa_prepare_fixed_rate(const cyfa_dims_t* dims, double rho, const float* decay_logit,
                            const float* beta_logit, const float* A, const double* lambda0,
                            float* lam_mod, float* g_cum, float* beta, double* lambda_end,
                            void* stream);

/*
 * cyfa_prepare_varlen -- cyfa_prepare for variable-length sequences packed into one stream:
 * dims.B = 1, dims.T the total token count, and sequence j (0 <= j < nseq) on tokens
 * [cu_seqlens[j], cu_seqlens[j+1]) (cu_seqlens: device int32 [nseq + 1], non-decreasing, from 0
 * to T; empty sequences are allowed).  Each sequence is the operator on its own: its clock
 * starts at lambda0[j,h] (lambda0 [nseq, H] fp64, nullable for 0) and its states at zero.
 *   lam_mod, beta  as in cyfa_prepare, the clock restarting at every sequence start.
 *   g_cum          as in cyfa_prepare, minus 64 for every sequence start s > 0 with
 *                  chunk_start(t) <= s <= t: every decay factor exp(g_t - g_s) of the chunk
 *                  form (App. B Eq. app-chunk-decay) that spans a start then carries exp(-64),
 *                  which removes every contribution of an earlier sequence in fp32, while the
 *                  factors inside a sequence keep their value (one extra fp32 rounding of g).
 *   lambda_end     [nseq, H] fp64 (nullable): each sequence's final clock.
 * clock_logit may be NULL: the fixed-rate clock delta = 1 / rho of cyfa_prepare_fixed_rate.
 * cyfa_chunk_fwd and cyfa_chunk_bwd take the results as they are (B = 1, T the total) and give
 * each sequence's outputs and gradients; the decay and clock gradients need no change because
 * every term that spans a sequence start vanishes with its decay factor.  Kbar0 / Vbar0 give the
 * first sequence's initial states; Kbar_out / Vbar_out receive the last sequence's final states
 * (the chunk calls export no per-sequence states).  T must still be a multiple of the chunk
 * (pad with one more sequence).  Needs cyfa_workspace_size(CYFA_WS_PREPARE_VARLEN) bytes.
 * Offsets that are not a non-decreasing cover of [0, T] are detected on the device: the next
 * cyfa_check() returns CYFA_ERR_ARG (the results are then meaningless).
 */
int cyfa_prepare_varlen(const cyfa_dims_t* dims, const int* cu_seqlens, int nseq,
                        const float* clock_logit, double rho, const float* decay_logit,
                        const float* beta_logit, const float* A, const double* lambda0,
                        float* lam_mod, float* g_cum, float* beta, double* lambda_end,
                        void* workspace, size_t workspace_bytes, void* stream);

/*
 * cyfa_prepare_noalloc -- cyfa_prepare for callers that cannot provide any device memory of
 * their own beyond the tensors (the paper has no counterpart: this is a deployment variant).
 * Typical such callers are a serving process or plugin host that reserves all device memory
 * up front through its own allocator and forbids later cudaMalloc calls, or a latency-critical
 * loop that must not allocate.  Arguments and results are those of cyfa_prepare, without the
 * workspace.  It calls no allocator: the per-segment partial sums live in one fixed array
 * compiled into the library (256 KiB of fp64, held on every GPU that loads the library until
 * the process exits), which limits B * H * ceil(T / 1024) to 32768; larger shapes return
 * CYFA_ERR_WORKSPACE before anything is launched.  The first call made on a device looks up
 * the array's device address (cudaGetSymbolAddress) with that device current; make that first
 * call before any stream capture.  The looked-up address is kept for the life of the process:
 * do not use this entry point after a cudaDeviceReset (or any other reset of the device's
 * primary context) in the same process, since the kept address may then be stale.  All calls
 * share the array and each call overwrites it entirely before reading it, so nothing needs
 * clearing, but calls that may run concurrently on the GPU (on different streams, or different
 * host threads) race on it and must not overlap.  Argument errors are those of cyfa_prepare.
 */
int cyfa_prepare_noalloc(const cyfa_dims_t* dims, const float* clock_logit,
                         const float* decay_logit, const float* beta_logit, const float* A,
                         const double* lambda0, float* lam_mod, float* g_cum, float* beta,
                         double* lambda_end, void* stream);

/*
 * cyfa_saved_size -- bytes of the forward intermediates that cyfa_chunk_fwd can save for
 * cyfa_chunk_bwd: the states [Kbar | Vbar] at the start of every chunk (App. B's
 * chunk-boundary states).  On the tensor-core kernels: every 128-token chunk, fp16,
 * [B*H][T/128][2][128][128] with the Fourier rows in the kernels' internal order, followed by
 * the fp16 readout matrix M = R Phi [H][128][128] (the backward then does not recompute it).  On the
 * CUDA-core kernels with 128 storage rows and a forward walking 64-token chunks (chunk 64, or
 * d = 256): every 64-token chunk, fp32, [B*H][T/64][128][2d] in the paper's row order.  0
 * otherwise (nothing is saved).  No paper counterpart beyond those states: this is the usual
 * activation-saving trade of a training step (HBM traffic for recomputation).
 */
int cyfa_saved_size(const cyfa_dims_t* dims, size_t* bytes);

/*
 * cyfa_chunk_fwd -- forward of the operator, chunk-wise two-pass form (Sec. 3.3 Eq.
 * cyfa-two-pass; App. B Eqs. app-cyfa-key-chunk, app-cyfa-value-chunk).
 * Inputs are the outputs of cyfa_prepare plus q, k, v and R.  Kbar0 / Vbar0 (nullable,
 * both or neither) give the states before token 0 in the same clock origin as lambda0.
 * o receives the output; Kbar_out / Vbar_out (nullable) receive the states after token T-1.
 * saved (nullable, device, 16-byte aligned, cyfa_saved_size bytes) receives the chunk-start
 * states for cyfa_chunk_bwd; ignored where cyfa_saved_size is 0.
 * The tensor-core kernels (bf16, d = 128) compute with fp16 operands (fp32 accumulation):
 * q, k, v must lie within fp16's range (|x| < 65504), and so must the states they build, whose
 * entries are bounded by 0.126 max|v| / (1 - max alpha) (|a_t| <= sqrt(2/m) beta_t entrywise;
 * a geometric sum of decays).  Where an fp16 snapshot of a state overflows anyway, the output o
 * becomes non-finite; the kernel that writes o then records CYFA_ERR_RANGE, which the next
 * cyfa_check() returns.  The CUDA-core kernels (fp32 throughout) have no such limit.
 */
int cyfa_chunk_fwd(const cyfa_dims_t* dims, const void* q, const void* k, const void* v,
                   const float* lam_mod, const float* g_cum, const float* beta, const float* R,
                   const float* Kbar0, const float* Vbar0, void* o, float* Kbar_out,
                   float* Vbar_out, void* saved, void* workspace, size_t workspace_bytes,
                   void* stream);

/*
 * cyfa_chunk_bwd -- gradient of sum(o * dO) with respect to q, k, v, the three logits, and
 * (nullable outputs) R and A, starting from zero state at token 0.  The clock gradient is
 * the reverse cumulative sum dL/d delta_s = sum_{t>=s} dL/d lambda_t of App. D.1 Eq.
 * app-clock-gradient-accumulation; the decay gradient is the reverse cumulative sum of
 * the per-token gradient of the cumulative log-decay.  dR [H,m,m] and dA [H] are sums
 * over the batch (dR through M = R Phi of the middle readout, Sec. 3.3 Eq. cyfa-two-pass).
 * Inputs are those of cyfa_chunk_fwd plus the raw clock / decay logits
 * and A (for the activation derivatives).  clock_logit and d_clock_logit are both NULL for a
 * fixed-rate clock (cyfa_prepare_fixed_rate): the clock gradient is then not formed.  saved (nullable): the buffer a cyfa_chunk_fwd call
 * with the same dims, inputs and no initial state filled; the chunk-start states are then
 * read from it instead of being recomputed.  Ignored where cyfa_saved_size is 0.
 * The tensor-core kernels' fp16 intermediates include the adjoint states (which grow with
 * |dO| / (1 - max alpha)) and dL/do' = Vbar dO per token (which grows with |v| |dO| / (1 -
 * max alpha)); all of them feed the three logit gradients, so an overflow anywhere makes one
 * of those non-finite, and the kernel that writes them then records CYFA_ERR_RANGE, which the
 * next cyfa_check() returns.
 */
int cyfa_chunk_bwd(const cyfa_dims_t* dims, const void* q, const void* k, const void* v,
                   const float* lam_mod, const float* g_cum, const float* beta, const float* R,
                   const float* clock_logit, const float* decay_logit, const float* A,
                   const void* dO, void* dq, void* dk, void* dv, float* d_clock_logit,
                   float* d_decay_logit, float* d_beta_logit, float* dR, float* dA,
                   const void* saved, void* workspace, size_t workspace_bytes, void* stream);

/*
 * cyfa_step -- one decode token for every (b, h), in place on the persistent state
 * (Sec. 3.2 Eq. cyfa-absolute-recurrence and Eq. cyfa-absolute-readout, one step).
 * q, k, v, o are [B, H, d] (dims.T is ignored); the logits are [B, H] fp32.
 * Kbar, Vbar [B, H, ms, d] fp32 (ms = 128 for m <= 127, 256 above) and lambda [B, H] fp64 are
 * read and overwritten.
 * Needs no workspace.
 */
int cyfa_step(const cyfa_dims_t* dims, const void* q, const void* k, const void* v,
              const float* clock_logit, const float* decay_logit, const float* beta_logit,
              const float* A, const float* R, float* Kbar, float* Vbar, double* lambda, void* o,
              void* stream);

/*
 * The mixer's neighbours of the operator (Sec. 3.4, Mixer and backbone: ShortConv on q, k, v,
 * RMSNorm of the queries and keys, head-wise RMSNorm of the output and a sigmoid output gate).
 * The paper gives no formulas for them; this library's reading, with every tensor [B, T, H, d]
 * in dims.dtype (channel c = h d + i), filters [H d][4] fp32 and gains [d] fp32 shared by the
 * heads:
 *   cyfa_mixer_pre:   a_t = silu(sum_{i<4} w[c][i] x_{t-3+i}[c])  (causal depthwise ShortConv,
 *                     width 4, zero before token 0, per batch row), then for q and k
 *                     q_t = a_t / sqrt(mean_d(a_t^2) + eps) * g per (token, head); v = a.
 *   cyfa_mixer_post:  y_t = o_t / sqrt(mean_d(o_t^2) + eps) * g * sigmoid(z_t), z the gate
 *                     logits of the mixer's low-rank gate projection.
 * The *_bwd calls give the gradients of sum(out * d_out) with respect to every input and
 * parameter (filter and gain gradients summed over the batch and, for gains, the heads);
 * they need cyfa_workspace_size(CYFA_WS_MIXER) bytes of workspace.  Tensor pointers must be
 * 16-byte aligned (CYFA_ERR_ALIGN otherwise).  The projections around
 * them are plain matrix products left to the caller.  dims is that of the operator call (T, H,
 * dk and dtype are used; m and chunk are checked as for the other calls).
 */
int cyfa_mixer_pre(const cyfa_dims_t* dims, const void* xq, const void* xk, const void* xv,
                   const float* wq, const float* wk, const float* wv, const float* gq,
                   const float* gk, float eps, void* q, void* k, void* v, void* stream);
int cyfa_mixer_pre_bwd(const cyfa_dims_t* dims, const void* xq, const void* xk, const void* xv,
                       const float* wq, const float* wk, const float* wv, const float* gq,
                       const float* gk, float eps, const void* dq, const void* dk, const void* dv,
                       void* dxq, void* dxk, void* dxv, float* dwq, float* dwk, float* dwv,
                       float* dgq, float* dgk, void* workspace, size_t workspace_bytes,
                       void* stream);
int cyfa_mixer_post(const cyfa_dims_t* dims, const void* o, const void* z, const float* g,
                    float eps, void* y, void* stream);
int cyfa_mixer_post_bwd(const cyfa_dims_t* dims, const void* o, const void* z, const float* g,
                        float eps, const void* dy, void* d_o, void* dz, float* dg,
                        void* workspace, size_t workspace_bytes, void* stream);

/*
 * cyfa_check -- wait for `stream`, then report (and clear) the device error words that the
 * kernels set: CYFA_ERR_TIMEOUT when a bounded device-side wait gave up, else CYFA_ERR_ARG when
 * cyfa_prepare_varlen found invalid sequence offsets, else CYFA_ERR_RANGE when a non-finite
 * value reached an output of the tensor-core kernels, else CYFA_ERR_CUDA when a CUDA-core chunk
 * kernel found its launch outside its shared-memory layout or block size (it then returned
 * without touching memory: an internal error), else CYFA_OK; CYFA_ERR_CUDA also if the stream
 * itself reports an error.
 */
int cyfa_check(void* stream);

/*
 * cyfa_selftest_mma -- self-check of the tensor-core (tcgen05 / TMEM / TMA) operand layouts the
 * chunk kernels rely on; the paper has no counterpart.  Computes D = op(X) op(Y) for row-major
 * bf16 X, Y [128 x 128] (device pointers, 16-byte aligned) into fp32 D [128 x 128]:
 * variant bit 0 selects op(X) = X^T (A operand MN-major) instead of X (K-major); bit 1 selects
 * op(Y) = Y (B operand MN-major) instead of Y^T (K-major); bit 2 writes the operand tiles with
 * threads instead of TMA.  Synchronises `stream`; CYFA_ERR_TIMEOUT if a bounded wait expired.
 */
int cyfa_selftest_mma(int variant, const void* X, const void* Y, float* D, void* stream);

/*
 * cyfa_selftest_timeout -- self-check of failure detection; the paper has no counterpart.  One
 * device thread waits on an mbarrier that nothing ever completes, with the same bounded wait the
 * kernels use (which gives up after 2 s) but a limit of `limit_us` microseconds (1 .. 10^6).
 * When the wait gives up the kernel records CYFA_ERR_TIMEOUT and returns normally, exactly as the
 * chunk kernels do, so the CUDA context stays usable.  `elapsed_ns` (device pointer to one
 * unsigned 64-bit value, or NULL) receives the time the wait took.  Synchronises `stream`.
 * Returns CYFA_ERR_TIMEOUT when the wait expired (the expected outcome), CYFA_OK if it did not,
 * CYFA_ERR_ARG for a limit out of range, CYFA_ERR_CUDA on a launch failure.
 */
int cyfa_selftest_timeout(unsigned int limit_us, unsigned long long* elapsed_ns, void* stream);

/*
 * Launch accounting (host side, process-wide).  Every kernel launch of the library increments
 * a counter kept per kernel name.  With cyfa_stats_timing(1) each launch is also bracketed by
 * CUDA events recorded on its own stream; the elapsed times are summed per kernel when read.
 *   cyfa_stats_reset   -- forget all counters and timings.
 *   cyfa_stats_timing  -- 1 to time every launch from now on, 0 to stop.
 *   cyfa_stats_get     -- entry `index` (0-based, in order of first launch): its kernel name
 *                         (copied into name[name_len], NUL-terminated), launches and total
 *                         milliseconds (waits for the recorded events).  CYFA_ERR_ARG past
 *                         the last entry.
 */
int cyfa_stats_reset(void);
int cyfa_stats_timing(int on);
int cyfa_stats_get(int index, char* name, int name_len, long long* launches, double* total_ms);

#ifdef __cplusplus
}
#endif

#endif /* CYFA_H */
