// Launch interface between the C ABI (cyfa_api.cu) and the kernel translation units.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stddef.h>

struct cyfa_dims;

namespace cyfa {

// Host-side check of a dims struct shared by every entry point: CYFA_OK, or the error code the
// entry point returns before launching anything (need_T: T and chunk are used by the call).
int check_dims(const ::cyfa_dims* d, bool need_T);

// Counts one launch of the named kernel and, when timing is on (cyfa_stats_timing), brackets it
// with CUDA events on its stream.  Construct immediately before the <<<>>> launch.
class LaunchScope {
  public:
    LaunchScope(const char* name, cudaStream_t st);
    ~LaunchScope();
    LaunchScope(const LaunchScope&) = delete;
    LaunchScope& operator=(const LaunchScope&) = delete;

  private:
    cudaStream_t stream_;
    int idx_ = 0;
    cudaEvent_t start_ = nullptr;
};

// Slot geometry: m active relative-time slots (odd, 1 <= m <= 255) in ms storage rows (128 for
// m <= 127, 256 above); the real Fourier basis of App. A.1 Eq. app-real-fourier has the DC row
// and (m-1)/2 cosine-sine pairs, b = [1/sqrt(m), sqrt(2/m), 0, sqrt(2/m), 0, ...]
// (Eq. app-b-explicit), and rows m..ms-1 stay zero.  The constants are formed once on the host.
struct Slots {
    int m, npair, ms;
    float fm, inv_m, two_over_m, inv_sqrt_m, sqrt2_over_m;
    float omega1;           // 2 pi / m, the rotation rate of pair 1
};
constexpr int MS_MAX = 256;   // largest number of storage rows
inline int storage_rows(int m) { return m <= 127 ? 128 : 256; }
inline Slots make_slots(int m) {
    Slots s;
    s.m = m;
    s.npair = (m - 1) / 2;
    s.ms = storage_rows(m);
    s.fm = (float)m;
    s.inv_m = 1.f / (float)m;
    s.two_over_m = 2.f / (float)m;
    s.inv_sqrt_m = (float)(1.0 / __builtin_sqrt((double)m));
    s.sqrt2_over_m = (float)__builtin_sqrt(2.0 / (double)m);
    s.omega1 = 6.283185307179586f / (float)m;
    return s;
}

// The same geometry as compile-time constants for m = 127 (the paper's setting): kernels
// templated on the slot type fold every constant; runtime Slots serve the other m.
struct Slots127 {
    static constexpr int m = 127, npair = 63, ms = 128;
    static constexpr float fm = 127.f, inv_m = 1.f / 127.f, two_over_m = 2.f / 127.f;
    static constexpr float inv_sqrt_m = 0.088735650941611f, sqrt2_over_m = 0.125491161809579f;
    static constexpr float omega1 = 6.283185307179586f / 127.f;
};

struct Shape {
    int B, T, H, D, C;      // batch, tokens, heads, head dim (dk == dv), chunk walked by a kernel
    int Cg;                 // chunk length the g_cum input is local to (the caller's chunk)
    float scale;
    bool bf16;
    Slots sl;               // active slots
    __host__ __device__ int nchunk() const { return T / C; }
};

// ---- prepare (prepare.cu) ----
struct PrepareArgs {
    Shape s;
    const float *clock_logit, *decay_logit, *beta_logit, *A;
    const double* lambda0;
    float *lam_mod, *g_cum, *beta;
    double* lambda_end;
    double* seg_sum;   // workspace [B*H][nseg]
};
constexpr int PREP_SEG = 1024;  // tokens per prepare block (multiple of every chunk size)
size_t prepare_workspace(const Shape& s);
cudaError_t launch_prepare(const PrepareArgs& a, cudaStream_t st);
// Packed sequences (prepare_varlen.cu): a.s.B == 1, sequence j on tokens [cu[j], cu[j+1]);
// lambda0 / lambda_end are [nseq][H]; rho > 0 and a.clock_logit == nullptr for a fixed-rate clock.
size_t prepare_varlen_workspace(const Shape& s);
cudaError_t launch_prepare_varlen(const PrepareArgs& a, const int* cu, int nseq, double rho,
                                  double* seg, cudaStream_t st);
// Fixed-rate clock delta = 1 / rho (no clock logits, no scan, no workspace).
cudaError_t launch_prepare_fixed_rate(const PrepareArgs& a, double rho, cudaStream_t st);
// Reads (and clears) the error word of the packed-sequence prepare; synchronises the stream.
cudaError_t prep_read_error(cudaStream_t st, int* err);

// ---- readout matrix M = R Phi and its transpose (chunk_simt.cu) ----
// R [H, m, m]; M, MT [H, ms, ms] with the rows and columns m..ms-1 zero.
cudaError_t launch_readout_matrix(int H, const float* R, float* M, float* MT, const Slots& sl,
                                  cudaStream_t st);

// ---- chunk forward / backward ----
struct FwdArgs {
    Shape s;
    const void *q, *k, *v;
    const float *lam, *g, *beta, *M, *MT;
    const float *Kbar0, *Vbar0;
    void* o;
    float *Kout, *Vout;
    float* states;      // workspace [B*H][nchunk][ms][2D]: chunk-start [Kbar | Vbar]
};
cudaError_t launch_fwd_simt(const FwdArgs& a, cudaStream_t st);
cudaError_t launch_state_simt(const FwdArgs& a, cudaStream_t st);  // state pass only

struct BwdArgs {
    Shape s;            // s.C is the backward's own chunk length
    const void *q, *k, *v, *dO;
    const float *lam, *g, *beta, *M, *MT;
    const float *clock_logit, *decay_logit, *A;
    void *dq, *dk, *dv;
    float *d_clock, *d_decay, *d_beta, *dA;
    float* states;      // [B*H][nchunk][ms][2D] chunk-start states
    bool states_given;  // states holds the forward's saved states: the state pass is skipped
    float* adj;         // [B*H][nchunk][ms][2D] adjoints of the chunk-end states
    float* o2;          // [B*H][T][ms] o'' per token
    float* do1;         // [B*H][T][ms] dL/do' per token
    float* tok;         // [4][B*T*H]: dG part 1, d lambda part 1, dG part 2 / d lambda part 2 / d beta
    double* seg;        // [2][B*H][nseg] reverse-scan partials
    double* dA_part;    // [B*H*nseg]
    // dR (nullable): per-token z, p, dy, dl of the middle readout (fp32 [B*H][T][ms], paper
    // order), the partial dM blocks [H][dm_splits][ms][ms] and the output [H][m][m]
    float *mZ, *mP, *mDY, *mDL;
    float *dM, *dR;
};
// dR[h] = dM[h] Phi^T over the m active slots from dm_split partial dM blocks [H][split][128][128]
// whose Fourier (column) index is in the tensor-core order (tc_order) or in the paper's order
// (m <= 127).
cudaError_t launch_dr_finalize(const float* dMp, int dm_split, int H, bool tc_order, float* dR,
                               const Slots& sl, cudaStream_t st);
constexpr int BWD_C = 64;       // chunk length used by the SIMT backward with 128 storage rows
constexpr int BWD_C256 = 32;    // ... and with 256 (the tiles of a 64-token chunk would not fit)
inline int bwd_chunk(const Slots& sl) { return sl.ms == 128 ? BWD_C : BWD_C256; }
// Token ranges the CUDA-core dR reduction splits each head's B*T tokens into: about four blocks
// per SM of the GB300's 152 over the (ms / 64)^2 tiles and H heads, at least 256 tokens per
// range, at most 64.  A function of the shape alone, so the workspace size is fixed by the dims.
inline int dm_splits(const Shape& s) {
    const long long tiles = (long long)(s.sl.ms / 64) * (s.sl.ms / 64) * s.H;
    long long n = (4 * 152 + tiles - 1) / tiles;
    const long long by_tokens = ((long long)s.B * s.T + 255) / 256;
    if (n > by_tokens) n = by_tokens;
    if (n > 64) n = 64;
    return n < 1 ? 1 : (int)n;
}
cudaError_t launch_bwd_simt(const BwdArgs& a, cudaStream_t st);
// Read (and clear) the launch-check error words of the CUDA-core chunk kernels (forward and
// backward translation units); synchronise the stream.
cudaError_t simt_fwd_read_error(cudaStream_t st, int* err);
cudaError_t simt_bwd_read_error(cudaStream_t st, int* err);
// reverse cumulative sums of the per-token scalars in a.tok and the logit gradients
cudaError_t launch_bwd_gates(const BwdArgs& a, cudaStream_t st);

// ---- tensor-core path (tc_*.cu) ----
// Encode a 16-bit (bf16, or fp16 with f16 = true) TMA tensor map with 128-byte swizzle (dims /
// strides innermost first; strides in bytes for dims 1..rank-1).  False if the driver entry
// point is missing or encoding fails.
bool make_tmap_bf16(CUtensorMap* map, const void* base, int rank, const unsigned long long* dims,
                    const unsigned long long* strides_bytes, const unsigned* box, bool f16 = false);
cudaError_t launch_selftest_mma(int variant, const void* X, const void* Y, float* D,
                                cudaStream_t st, int* host_err);
// One thread waits on an mbarrier nothing arrives on with the kernels' own bounded wait, given a
// limit of limit_us; *host_err = CYFA_ERR_TIMEOUT when it gave up (synchronises st).
cudaError_t launch_timeout_probe(unsigned limit_us, unsigned long long* elapsed_ns,
                                 cudaStream_t st, int* host_err);

struct TcFwdArgs {
    Shape s;
    const float *lam, *g, *beta;
    const float *Kbar0, *Vbar0;   // nullable initial states [B,H,128,128]
    float *Kout, *Vout;           // nullable final states
    void* o;                      // bf16 [B,T,H,128]
    float* segS;                  // [B*H][nseg][128][256]: segment deltas, then segment-start states
    float* segG;                  // [B*H][nseg] total log-decay of each segment
    const __half* Mb;             // [H][128][128] fp16 M = R Phi
    __half* snap;                 // nullable [B*H][T/128][2][128][128] fp16: Kbar, Vbar at
                                  // each chunk start, written for the backward
    int nseg;
};
bool tc_fwd_supported(const Shape& s);
int tc_fwd_segments(const Shape& s);
cudaError_t launch_fwd_tc(const TcFwdArgs& a, const void* q, const void* k, const void* v,
                          cudaStream_t st);
// M = R Phi as fp16 in the tensor-core column order ([H][128][128], padding row / column zero).
cudaError_t launch_readout_f16(int H, const float* R, __half* Mb, const Slots& sl,
                               cudaStream_t st);
// Reads (and clears) the error word of the tensor-core kernels; synchronises the stream.
cudaError_t tc_read_error(cudaStream_t st, int* err);
cudaError_t tc_bwd_read_error(cudaStream_t st, int* err);
// TMA maps of [B, T, H, 128] bf16 tensors (boxes of box_rows tokens of one head) and of
// row-major [rows x 128] 16-bit arrays (box_rows-row boxes); null outputs are skipped.
bool tc_qkv_maps(const Shape& s, const void* q, const void* k, const void* v, CUtensorMap* mq,
                 CUtensorMap* mk, CUtensorMap* mv, unsigned box_rows = 128);
bool tc_rows_map(CUtensorMap* map, const void* base, unsigned long long rows, bool f16 = false,
                 unsigned box_rows = 128);
// Segment state contributions and the segment scan.
cudaError_t launch_fwd_segment_states(const TcFwdArgs& a, const void* k, const void* v,
                                      cudaStream_t st);
// The total log-decay of every segment, without the states.
cudaError_t launch_segment_decay(const TcFwdArgs& a, cudaStream_t st);

struct TcBwdArgs {
    Shape s;
    const float *lam, *g, *beta;
    float* segS;                 // forward segment-start states (tensor-core row order)
    float* segG;                 // total log-decay per segment
    float* segD;                 // adjoint: per-segment contributions, then end-of-segment adjoints
    int nseg;
    __half* snapF;               // [B*H][T/128][2][128][128] fp16: Kbar, Vbar at each chunk start
    bool saved;                  // snapF holds the forward's saved states: no recomputation
    __half* snapA;               // [B*H][T/128][2][128][128] fp16: D^K, D^V at each chunk end
    __half* O2;                  // [B*H][T][128] fp16: o'' (tensor-core order)
    __half* DO1;                 // [B*H][T][128] fp16: dL/do' (tensor-core order)
    const __half* Mb;            // [H][128][128] fp16 M = R Phi
    const void *q, *k;           // [B,T,H,128] bf16 (row reads of the epilogues)
    void *dq, *dk, *dv;
    float* tok;                  // [7][B*T*H] per-token scalars: row side of dG, d lambda;
                                 // intra-chunk column side of dG, d lambda; d beta;
                                 // inter-chunk column side of dG, d lambda
    float* bnd;                  // [B*H][T/128][2]: gamma^C <D, S>, gamma^C <D, Omega S>
    const float *clock_logit, *decay_logit, *A;
    float *d_clock, *d_decay, *d_beta, *dA;
    double* dA_part;             // [B*H][T/128]
    // dR (nullable): per-token z, p, dy, dl of the middle readout (fp16 [B*H][T][128]: z, dy in
    // the kernels' Fourier order, p, dl over the slots), per-head partial dM and the output
    __half *mZ, *mP, *mDY, *mDL;
    float* dMp;                  // [H][dm_split][128][128]
    int dm_split;
    float* dR;                   // [H][127][127]
};
cudaError_t launch_bwd_tc(const TcBwdArgs& a, const TcFwdArgs& f, const void* q, const void* k,
                          const void* v, const void* dO, cudaStream_t st);

// ---- mixer neighbours (mixer.cu) ----
// Arrays of three are (q, k, v); of two (q, k).
size_t mixer_workspace(const Shape& s);
cudaError_t launch_mixer_pre(const Shape& s, const void* const* x, const float* const* w,
                             const float* const* g, float eps, void* const* y, cudaStream_t st);
cudaError_t launch_mixer_pre_bwd(const Shape& s, const void* const* x, const float* const* w,
                                 const float* const* g, float eps, const void* const* dy,
                                 void* const* dx, float* const* dw, float* const* dg, void* ws,
                                 cudaStream_t st);
cudaError_t launch_mixer_post(const Shape& s, const void* o, const void* z, const float* g,
                              float eps, void* y, cudaStream_t st);
cudaError_t launch_mixer_post_bwd(const Shape& s, const void* o, const void* z, const float* g,
                                  float eps, const void* dy, void* dO, void* dz, float* dg,
                                  void* ws, cudaStream_t st);

// ---- decode (decode.cu) ----
struct StepArgs {
    int B, H, D;
    Slots sl;
    float scale;
    bool bf16;
    const void *q, *k, *v;
    const float *clock_logit, *decay_logit, *beta_logit, *A, *R;
    float *Kbar, *Vbar;
    double* lambda;
    void* o;
};
cudaError_t launch_step(const StepArgs& a, cudaStream_t st);

}  // namespace cyfa
