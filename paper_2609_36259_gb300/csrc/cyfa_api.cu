// C ABI of the CyFA operator: argument checking, workspace layout, and launches on the
// caller's stream.  The declarations and their contracts are in include/cyfa.h.
#include <stdint.h>

#include "../../include/cyfa.h"
#include "common.cuh"
#include "kernels.h"

using namespace cyfa;

namespace {

constexpr size_t ALIGN = 256;
inline size_t up(size_t x) { return (x + ALIGN - 1) / ALIGN * ALIGN; }

// Sequential carve-out of a workspace buffer.
struct Carver {
    char* base;
    size_t off = 0;
    template <typename T>
    T* take(size_t count) {
        T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
        off += up(count * sizeof(T));
        return p;
    }
};

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

// The (b, h) sequences go on gridDim.y of the per-sequence launches, whose limit is 65535.
constexpr long long kMaxSequences = 65535;

int cyfa::check_dims(const cyfa_dims_t* d, bool need_T) {
    if (!d) return CYFA_ERR_ARG;
    if (d->B <= 0 || d->H <= 0 || d->dk <= 0 || d->dv <= 0 || (need_T && d->T <= 0))
        return CYFA_ERR_ARG;
    if (d->dtype != CYFA_DTYPE_BF16 && d->dtype != CYFA_DTYPE_FP32) return CYFA_ERR_ARG;
    // m: odd, 1..255 (128 storage rows up to 127, 256 above)
    if (d->m < 1 || d->m > 255 || d->m % 2 == 0) return CYFA_ERR_SHAPE;
    if (d->dk != d->dv || (d->dk != 64 && d->dk != 128 && d->dk != 256)) return CYFA_ERR_SHAPE;
    if ((long long)d->B * d->H > kMaxSequences) return CYFA_ERR_SHAPE;
    if (need_T) {
        if (d->chunk != 64 && d->chunk != 128) return CYFA_ERR_SHAPE;
        if (d->T % d->chunk != 0) return CYFA_ERR_SHAPE;
    }
    return CYFA_OK;
}

namespace {

Shape shape_of(const cyfa_dims_t* d) {
    Shape s;
    s.B = d->B;
    s.T = d->T;
    s.H = d->H;
    s.D = d->dk;
    s.C = d->chunk;
    s.Cg = d->chunk;
    s.scale = d->scale;
    s.bf16 = d->dtype == CYFA_DTYPE_BF16;
    s.sl = make_slots(d->m);
    return s;
}

// The tensor-core kernels hold 128 storage rows.
bool use_tc(const cyfa_dims_t* d, const Shape& s) {
    return !(d->flags & CYFA_FLAG_CUDA_CORES) && s.sl.ms == 128 && tc_fwd_supported(s);
}

// The CUDA-core forward walks the caller's chunk, except at d = 256 or with 256 storage rows,
// where it walks 64-token chunks (its register and shared tiles of a 128-token chunk would not
// fit); g_cum stays local to the caller's chunk (Cg) and the kernels rebase it.
Shape simt_fwd_shape(Shape s) {
    if (s.D == 256 || s.sl.ms == 256) s.C = 64;
    return s;
}

struct FwdLayout {
    float *M, *MT, *states;          // CUDA-core path
    float *segS, *segG;              // tensor-core path
    __half* Mb;
    int nseg;
    size_t bytes;
};
FwdLayout fwd_layout(const Shape& s0, bool tc_path, void* ws) {
    const Shape s = tc_path ? s0 : simt_fwd_shape(s0);
    const size_t ms = s.sl.ms;
    Carver c{static_cast<char*>(ws)};
    FwdLayout L{};
    L.M = c.take<float>((size_t)s.H * ms * ms);
    L.MT = c.take<float>((size_t)s.H * ms * ms);
    if (tc_path) {
        L.nseg = tc_fwd_segments(s);
        L.Mb = c.take<__half>((size_t)s.H * MS * MS);
        L.segS = c.take<float>((size_t)s.B * s.H * L.nseg * MS * 256);
        L.segG = c.take<float>((size_t)s.B * s.H * L.nseg);
    } else {
        L.states = c.take<float>((size_t)s.B * s.H * s.nchunk() * ms * 2 * s.D);
    }
    L.bytes = c.off;
    return L;
}

struct BwdLayout {
    float *M, *MT, *states, *adj, *o2, *do1, *tok;     // CUDA-core path (+ shared M, tok)
    double *seg, *dA_part;
    __half *Mb, *snapF, *snapA, *O2b, *DO1b;   // tensor-core path (fp16 operands)
    float *segS, *segG, *segD, *bnd;
    double* dA_chunk;
    __half *mZ, *mP, *mDY, *mDL;     // middle-readout vectors for dR
    float *fZ, *fP, *fDY, *fDL, *fdM;   // the same on the CUDA-core path (fp32)
    float* dMp;
    int dm_split;
    int nseg;
    size_t bytes;
};
BwdLayout bwd_layout(const Shape& s0, bool tc_path, void* ws) {
    Shape s = s0;
    s.C = bwd_chunk(s.sl);
    const size_t ms = s.sl.ms;
    Carver c{static_cast<char*>(ws)};
    BwdLayout L{};
    const size_t BH = (size_t)s.B * s.H;
    const size_t nseg = (s.T + PREP_SEG - 1) / PREP_SEG;
    L.M = c.take<float>((size_t)s.H * ms * ms);
    L.MT = c.take<float>((size_t)s.H * ms * ms);
    L.tok = c.take<float>((tc_path ? 7 : 5) * BH * s.T);
    L.seg = c.take<double>(2 * BH * nseg);
    L.dA_part = c.take<double>(BH * nseg);
    if (tc_path) {
        const size_t nct = s.T / 128;
        L.nseg = tc_fwd_segments(s0);
        L.Mb = c.take<__half>((size_t)s.H * MS * MS);
        L.segS = c.take<float>(BH * L.nseg * MS * 256);
        L.segD = c.take<float>(BH * L.nseg * MS * 256);
        L.segG = c.take<float>(BH * L.nseg);
        L.snapF = c.take<__half>(BH * nct * 2 * MS * 128);
        L.snapA = c.take<__half>(BH * nct * 2 * MS * 128);
        L.O2b = c.take<__half>(BH * s.T * MS);
        L.DO1b = c.take<__half>(BH * s.T * MS);
        L.bnd = c.take<float>(BH * nct * 2);
        L.dA_chunk = c.take<double>(BH * nct);
        L.mZ = c.take<__half>(BH * s.T * MS);
        L.mP = c.take<__half>(BH * s.T * MS);
        L.mDY = c.take<__half>(BH * s.T * MS);
        L.mDL = c.take<__half>(BH * s.T * MS);
        const size_t nch = (size_t)s.B * nct;
        L.dm_split = (int)(nch < 32 ? nch : 32);
        L.dMp = c.take<float>((size_t)s.H * L.dm_split * MS * MS);
    } else {
        L.states = c.take<float>(BH * s.nchunk() * ms * 2 * s.D);
        L.adj = c.take<float>(BH * s.nchunk() * ms * 2 * s.D);
        L.o2 = c.take<float>(BH * s.T * ms);
        L.do1 = c.take<float>(BH * s.T * ms);
        L.fZ = c.take<float>(BH * s.T * ms);
        L.fP = c.take<float>(BH * s.T * ms);
        L.fDY = c.take<float>(BH * s.T * ms);
        L.fDL = c.take<float>(BH * s.T * ms);
        L.fdM = c.take<float>((size_t)s.H * dm_splits(s) * ms * ms);
    }
    L.bytes = c.off;
    return L;
}

inline int cuda_status(cudaError_t e) { return e == cudaSuccess ? CYFA_OK : CYFA_ERR_CUDA; }

}  // namespace

extern "C" {

int cyfa_version(void) { return 100; }

const char* cyfa_error_string(int code) {
    switch (code) {
        case CYFA_OK: return "ok";
        case CYFA_ERR_ARG: return "invalid argument (null pointer or non-positive size)";
        case CYFA_ERR_SHAPE: return "unsupported shape (m odd in 1..255, dk == dv in {64,128,256}, chunk in {64,128}, T % chunk == 0, B*H <= 65535)";
        case CYFA_ERR_ALIGN: return "tensor pointer not 16-byte aligned";
        case CYFA_ERR_WORKSPACE: return "workspace missing or too small";
        case CYFA_ERR_CUDA: return "CUDA runtime error";
        case CYFA_ERR_TIMEOUT: return "bounded device-side wait expired";
        case CYFA_ERR_UNSUPPORTED: return "request not implemented by this build";
        case CYFA_ERR_RANGE: return "non-finite result: an fp16 operand of the tensor-core kernels overflowed, or an input was not finite";
        default: return "unknown cyfa error code";
    }
}

int cyfa_workspace_size(const cyfa_dims_t* dims, int which, size_t* bytes) {
    if (!bytes) return CYFA_ERR_ARG;
    const int rc = check_dims(dims, true);
    if (rc) return rc;
    const Shape s = shape_of(dims);
    switch (which) {
        case CYFA_WS_PREPARE: *bytes = up(prepare_workspace(s)); return CYFA_OK;
        case CYFA_WS_PREPARE_VARLEN: *bytes = up(prepare_varlen_workspace(s)); return CYFA_OK;
        case CYFA_WS_MIXER: *bytes = up(mixer_workspace(s)); return CYFA_OK;
        case CYFA_WS_FWD: *bytes = fwd_layout(s, use_tc(dims, s), nullptr).bytes; return CYFA_OK;
        case CYFA_WS_BWD: *bytes = bwd_layout(s, use_tc(dims, s), nullptr).bytes; return CYFA_OK;
        default: return CYFA_ERR_ARG;
    }
}

// Tensor-core path: fp16 chunk-start states [B*H][T/128][2][128][128], then the fp16 readout
// matrix M = R Phi [H][128][128] the forward computed (the backward reads it instead of
// recomputing it).  The states' size is a multiple of 64 KiB, so M stays aligned.
size_t saved_state_bytes(const Shape& s) {
    return (size_t)s.B * s.H * (s.T / 128) * 2 * 128 * 128 * 2;
}
size_t saved_bytes(const Shape& s) { return saved_state_bytes(s) + (size_t)s.H * MS * MS * 2; }
__half* saved_mb(const Shape& s, const void* saved) {
    return reinterpret_cast<__half*>(static_cast<char*>(const_cast<void*>(saved)) +
                                     saved_state_bytes(s));
}

// The CUDA-core backward can read the forward's fp32 chunk-start states where both walk the same
// chunks (128 storage rows, and a forward of 64-token chunks: caller chunk 64, or d = 256).
bool simt_saved_ok(const Shape& s) {
    return s.sl.ms == 128 && simt_fwd_shape(s).C == bwd_chunk(s.sl);
}
// fp32 chunk-start blocks [B*H][T/64][128][2d] of the CUDA-core path
size_t saved_bytes_simt(const Shape& s) {
    return (size_t)s.B * s.H * (s.T / BWD_C) * 128 * 2 * s.D * sizeof(float);
}
size_t saved_size_of(const cyfa_dims_t* d, const Shape& s) {
    if (use_tc(d, s)) return saved_bytes(s);
    return simt_saved_ok(s) ? saved_bytes_simt(s) : 0;
}

int cyfa_saved_size(const cyfa_dims_t* dims, size_t* bytes) {
    if (!bytes) return CYFA_ERR_ARG;
    const int rc = check_dims(dims, true);
    if (rc) return rc;
    const Shape s = shape_of(dims);
    *bytes = saved_size_of(dims, s);
    return CYFA_OK;
}

int cyfa_prepare(const cyfa_dims_t* dims, const float* clock_logit, const float* decay_logit,
                 const float* beta_logit, const float* A, const double* lambda0, float* lam_mod,
                 float* g_cum, float* beta, double* lambda_end, void* workspace,
                 size_t workspace_bytes, void* stream) {
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (!clock_logit || !decay_logit || !beta_logit || !A || !lam_mod || !g_cum || !beta)
        return CYFA_ERR_ARG;
    const Shape s = shape_of(dims);
    if (!workspace || workspace_bytes < prepare_workspace(s)) return CYFA_ERR_WORKSPACE;
    PrepareArgs a;
    a.s = s;
    a.clock_logit = clock_logit;
    a.decay_logit = decay_logit;
    a.beta_logit = beta_logit;
    a.A = A;
    a.lambda0 = lambda0;
    a.lam_mod = lam_mod;
    a.g_cum = g_cum;
    a.beta = beta;
    a.lambda_end = lambda_end;
    a.seg_sum = static_cast<double*>(workspace);
    return cuda_status(launch_prepare(a, static_cast<cudaStream_t>(stream)));
}

int cyfa_prepare_fixed_rate(const cyfa_dims_t* dims, double rho, const float* decay_logit,
                            const float* beta_logit, const float* A, const double* lambda0,
                            float* lam_mod, float* g_cum, float* beta, double* lambda_end,
                            void* stream) {
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (!(rho > 0.0) || !decay_logit || !beta_logit || !A || !lam_mod || !g_cum || !beta)
        return CYFA_ERR_ARG;
    PrepareArgs a{};
    a.s = shape_of(dims);
    a.clock_logit = nullptr;
    a.decay_logit = decay_logit;
    a.beta_logit = beta_logit;
    a.A = A;
    a.lambda0 = lambda0;
    a.lam_mod = lam_mod;
    a.g_cum = g_cum;
    a.beta = beta;
    a.lambda_end = lambda_end;
    return cuda_status(launch_prepare_fixed_rate(a, rho, static_cast<cudaStream_t>(stream)));
}

int cyfa_prepare_varlen(const cyfa_dims_t* dims, const int* cu_seqlens, int nseq,
                        const float* clock_logit, double rho, const float* decay_logit,
                        const float* beta_logit, const float* A, const double* lambda0,
                        float* lam_mod, float* g_cum, float* beta, double* lambda_end,
                        void* workspace, size_t workspace_bytes, void* stream) {
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (dims->B != 1 || nseq <= 0 || !cu_seqlens) return CYFA_ERR_ARG;
    if (!clock_logit && !(rho > 0.0)) return CYFA_ERR_ARG;
    if (!decay_logit || !beta_logit || !A || !lam_mod || !g_cum || !beta) return CYFA_ERR_ARG;
    const Shape s = shape_of(dims);
    if (!workspace || workspace_bytes < prepare_varlen_workspace(s)) return CYFA_ERR_WORKSPACE;
    PrepareArgs a{};
    a.s = s;
    a.clock_logit = clock_logit;
    a.decay_logit = decay_logit;
    a.beta_logit = beta_logit;
    a.A = A;
    a.lambda0 = lambda0;
    a.lam_mod = lam_mod;
    a.g_cum = g_cum;
    a.beta = beta;
    a.lambda_end = lambda_end;
    return cuda_status(launch_prepare_varlen(a, cu_seqlens, nseq, clock_logit ? 1.0 : rho,
                                             static_cast<double*>(workspace),
                                             static_cast<cudaStream_t>(stream)));
}

int cyfa_chunk_fwd(const cyfa_dims_t* dims, const void* q, const void* k, const void* v,
                   const float* lam_mod, const float* g_cum, const float* beta, const float* R,
                   const float* Kbar0, const float* Vbar0, void* o, float* Kbar_out,
                   float* Vbar_out, void* saved, void* workspace, size_t workspace_bytes,
                   void* stream) {
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (!q || !k || !v || !lam_mod || !g_cum || !beta || !R || !o) return CYFA_ERR_ARG;
    if ((Kbar0 == nullptr) != (Vbar0 == nullptr)) return CYFA_ERR_ARG;
    if ((Kbar_out == nullptr) != (Vbar_out == nullptr)) return CYFA_ERR_ARG;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o)) return CYFA_ERR_ALIGN;
    if ((Kbar0 && (!aligned16(Kbar0) || !aligned16(Vbar0))) ||
        (Kbar_out && (!aligned16(Kbar_out) || !aligned16(Vbar_out))))
        return CYFA_ERR_ALIGN;
    const Shape s = shape_of(dims);
    const bool tc_path = use_tc(dims, s);
    if (saved && !aligned16(saved)) return CYFA_ERR_ALIGN;
    const FwdLayout need = fwd_layout(s, tc_path, nullptr);
    if (!workspace || workspace_bytes < need.bytes) return CYFA_ERR_WORKSPACE;
    if (!aligned16(workspace)) return CYFA_ERR_ALIGN;
    const FwdLayout L = fwd_layout(s, tc_path, workspace);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // with saved states on, M goes next to them for the backward
    __half* Mb = (tc_path && saved) ? saved_mb(s, saved) : L.Mb;
    rc = cuda_status(tc_path ? launch_readout_f16(s.H, R, Mb, s.sl, st)
                             : launch_readout_matrix(s.H, R, L.M, L.MT, s.sl, st));
    if (rc) return rc;
    if (tc_path) {
        TcFwdArgs t;
        t.s = s;
        t.lam = lam_mod;
        t.g = g_cum;
        t.beta = beta;
        t.Kbar0 = Kbar0;
        t.Vbar0 = Vbar0;
        t.Kout = Kbar_out;
        t.Vout = Vbar_out;
        t.o = o;
        t.segS = L.segS;
        t.segG = L.segG;
        t.Mb = Mb;
        t.snap = static_cast<__half*>(saved);
        t.nseg = L.nseg;
        return cuda_status(launch_fwd_tc(t, q, k, v, st));
    }
    FwdArgs a;
    a.s = simt_fwd_shape(s);
    a.q = q;
    a.k = k;
    a.v = v;
    a.lam = lam_mod;
    a.g = g_cum;
    a.beta = beta;
    a.M = L.M;
    a.MT = L.MT;
    a.Kbar0 = Kbar0;
    a.Vbar0 = Vbar0;
    a.o = o;
    a.Kout = Kbar_out;
    a.Vout = Vbar_out;
    // the chunk-start states go to the caller's buffer when it keeps them for the backward
    a.states = (saved && simt_saved_ok(s)) ? static_cast<float*>(saved) : L.states;
    return cuda_status(launch_fwd_simt(a, st));
}

int cyfa_chunk_bwd(const cyfa_dims_t* dims, const void* q, const void* k, const void* v,
                   const float* lam_mod, const float* g_cum, const float* beta, const float* R,
                   const float* clock_logit, const float* decay_logit, const float* A,
                   const void* dO, void* dq, void* dk, void* dv, float* d_clock_logit,
                   float* d_decay_logit, float* d_beta_logit, float* dR, float* dA,
                   const void* saved, void* workspace, size_t workspace_bytes, void* stream) {
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (!q || !k || !v || !lam_mod || !g_cum || !beta || !R || !decay_logit || !A || !dO || !dq ||
        !dk || !dv || !d_decay_logit || !d_beta_logit)
        return CYFA_ERR_ARG;
    // both or neither: a fixed-rate clock has no clock logits and no clock gradient
    if ((clock_logit == nullptr) != (d_clock_logit == nullptr)) return CYFA_ERR_ARG;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(dO) || !aligned16(dq) ||
        !aligned16(dk) || !aligned16(dv))
        return CYFA_ERR_ALIGN;
    if (saved && !aligned16(saved)) return CYFA_ERR_ALIGN;
    const Shape s = shape_of(dims);
    const bool tc_path = use_tc(dims, s);
    const BwdLayout need = bwd_layout(s, tc_path, nullptr);
    if (!workspace || workspace_bytes < need.bytes) return CYFA_ERR_WORKSPACE;
    if (!aligned16(workspace)) return CYFA_ERR_ALIGN;
    const BwdLayout L = bwd_layout(s, tc_path, workspace);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // the tensor-core path reads M from the saved buffer when the forward kept it there
    __half* Mb = (tc_path && saved) ? saved_mb(s, saved) : L.Mb;
    if (!(tc_path && saved)) {
        rc = cuda_status(tc_path ? launch_readout_f16(s.H, R, Mb, s.sl, st)
                                 : launch_readout_matrix(s.H, R, L.M, L.MT, s.sl, st));
        if (rc) return rc;
    }
    BwdArgs a{};
    a.s = s;
    a.s.C = bwd_chunk(s.sl);
    a.q = q;
    a.k = k;
    a.v = v;
    a.dO = dO;
    a.lam = lam_mod;
    a.g = g_cum;
    a.beta = beta;
    a.M = L.M;
    a.MT = L.MT;
    a.clock_logit = clock_logit;
    a.decay_logit = decay_logit;
    a.A = A;
    a.dq = dq;
    a.dk = dk;
    a.dv = dv;
    a.d_clock = d_clock_logit;
    a.d_decay = d_decay_logit;
    a.d_beta = d_beta_logit;
    a.dA = dA;
    a.states_given = !tc_path && saved && simt_saved_ok(s);
    a.states = a.states_given ? static_cast<float*>(const_cast<void*>(saved)) : L.states;
    a.adj = L.adj;
    a.o2 = L.o2;
    a.do1 = L.do1;
    a.tok = L.tok;
    a.seg = L.seg;
    a.dA_part = L.dA_part;
    a.dR = tc_path ? nullptr : dR;
    a.mZ = (dR && !tc_path) ? L.fZ : nullptr;
    a.mP = (dR && !tc_path) ? L.fP : nullptr;
    a.mDY = (dR && !tc_path) ? L.fDY : nullptr;
    a.mDL = (dR && !tc_path) ? L.fDL : nullptr;
    a.dM = L.fdM;
    if (tc_path) {
        TcFwdArgs f{};
        f.s = s;
        f.lam = lam_mod;
        f.g = g_cum;
        f.beta = beta;
        f.segS = L.segS;
        f.segG = L.segG;
        f.Mb = Mb;
        f.snap = nullptr;
        f.nseg = L.nseg;
        TcBwdArgs t{};
        t.s = s;
        t.lam = lam_mod;
        t.g = g_cum;
        t.beta = beta;
        t.segS = L.segS;
        t.segG = L.segG;
        t.segD = L.segD;
        t.nseg = L.nseg;
        t.snapF = saved ? static_cast<__half*>(const_cast<void*>(saved)) : L.snapF;
        t.saved = saved != nullptr;
        t.snapA = L.snapA;
        t.O2 = L.O2b;
        t.DO1 = L.DO1b;
        t.Mb = Mb;
        t.q = q;
        t.k = k;
        t.dq = dq;
        t.dk = dk;
        t.dv = dv;
        t.tok = L.tok;
        t.bnd = L.bnd;
        t.clock_logit = clock_logit;
        t.decay_logit = decay_logit;
        t.A = A;
        t.d_clock = d_clock_logit;
        t.d_decay = d_decay_logit;
        t.d_beta = d_beta_logit;
        t.dA = dA;
        t.dA_part = L.dA_chunk;
        t.dR = dR;
        t.mZ = dR ? L.mZ : nullptr;
        t.mP = dR ? L.mP : nullptr;
        t.mDY = dR ? L.mDY : nullptr;
        t.mDL = dR ? L.mDL : nullptr;
        t.dMp = L.dMp;
        t.dm_split = L.dm_split;
        return cuda_status(launch_bwd_tc(t, f, q, k, v, dO, st));
    }
    return cuda_status(launch_bwd_simt(a, st));
}

int cyfa_step(const cyfa_dims_t* dims, const void* q, const void* k, const void* v,
              const float* clock_logit, const float* decay_logit, const float* beta_logit,
              const float* A, const float* R, float* Kbar, float* Vbar, double* lambda, void* o,
              void* stream) {
    int rc = check_dims(dims, false);
    if (rc) return rc;
    if (!q || !k || !v || !clock_logit || !decay_logit || !beta_logit || !A || !R || !Kbar ||
        !Vbar || !lambda || !o)
        return CYFA_ERR_ARG;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(Kbar) ||
        !aligned16(Vbar))
        return CYFA_ERR_ALIGN;
    StepArgs a;
    a.B = dims->B;
    a.H = dims->H;
    a.D = dims->dk;
    a.scale = dims->scale;
    a.bf16 = dims->dtype == CYFA_DTYPE_BF16;
    a.sl = make_slots(dims->m);
    a.q = q;
    a.k = k;
    a.v = v;
    a.clock_logit = clock_logit;
    a.decay_logit = decay_logit;
    a.beta_logit = beta_logit;
    a.A = A;
    a.R = R;
    a.Kbar = Kbar;
    a.Vbar = Vbar;
    a.lambda = lambda;
    a.o = o;
    return cuda_status(launch_step(a, static_cast<cudaStream_t>(stream)));
}

int cyfa_mixer_pre(const cyfa_dims_t* dims, const void* xq, const void* xk, const void* xv,
                   const float* wq, const float* wk, const float* wv, const float* gq,
                   const float* gk, float eps, void* q, void* k, void* v, void* stream) {
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (!xq || !xk || !xv || !wq || !wk || !wv || !gq || !gk || !q || !k || !v) return CYFA_ERR_ARG;
    if (!(eps >= 0.f)) return CYFA_ERR_ARG;
    for (const void* p : {xq, xk, xv, (const void*)q, (const void*)k, (const void*)v})
        if (!aligned16(p)) return CYFA_ERR_ALIGN;
    const void* x[3] = {xq, xk, xv};
    const float* w[3] = {wq, wk, wv};
    const float* g[2] = {gq, gk};
    void* y[3] = {q, k, v};
    return cuda_status(launch_mixer_pre(shape_of(dims), x, w, g, eps, y,
                                        static_cast<cudaStream_t>(stream)));
}

int cyfa_mixer_pre_bwd(const cyfa_dims_t* dims, const void* xq, const void* xk, const void* xv,
                       const float* wq, const float* wk, const float* wv, const float* gq,
                       const float* gk, float eps, const void* dq, const void* dk, const void* dv,
                       void* dxq, void* dxk, void* dxv, float* dwq, float* dwk, float* dwv,
                       float* dgq, float* dgk, void* workspace, size_t workspace_bytes,
                       void* stream) {
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (!xq || !xk || !xv || !wq || !wk || !wv || !gq || !gk || !dq || !dk || !dv || !dxq ||
        !dxk || !dxv || !dwq || !dwk || !dwv || !dgq || !dgk)
        return CYFA_ERR_ARG;
    if (!(eps >= 0.f)) return CYFA_ERR_ARG;
    for (const void* p : {xq, xk, xv, dq, dk, dv, (const void*)dxq, (const void*)dxk,
                          (const void*)dxv})
        if (!aligned16(p)) return CYFA_ERR_ALIGN;
    const Shape s = shape_of(dims);
    if (!workspace || workspace_bytes < mixer_workspace(s)) return CYFA_ERR_WORKSPACE;
    const void* x[3] = {xq, xk, xv};
    const float* w[3] = {wq, wk, wv};
    const float* g[2] = {gq, gk};
    const void* dy[3] = {dq, dk, dv};
    void* dx[3] = {dxq, dxk, dxv};
    float* dw[3] = {dwq, dwk, dwv};
    float* dg[2] = {dgq, dgk};
    return cuda_status(launch_mixer_pre_bwd(s, x, w, g, eps, dy, dx, dw, dg, workspace,
                                            static_cast<cudaStream_t>(stream)));
}

int cyfa_mixer_post(const cyfa_dims_t* dims, const void* o, const void* z, const float* g,
                    float eps, void* y, void* stream) {
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (!o || !z || !g || !y || !(eps >= 0.f)) return CYFA_ERR_ARG;
    if (!aligned16(o) || !aligned16(z) || !aligned16(y)) return CYFA_ERR_ALIGN;
    return cuda_status(launch_mixer_post(shape_of(dims), o, z, g, eps, y,
                                         static_cast<cudaStream_t>(stream)));
}

int cyfa_mixer_post_bwd(const cyfa_dims_t* dims, const void* o, const void* z, const float* g,
                        float eps, const void* dy, void* d_o, void* dz, float* dg,
                        void* workspace, size_t workspace_bytes, void* stream) {
    int rc = check_dims(dims, true);
    if (rc) return rc;
    if (!o || !z || !g || !dy || !d_o || !dz || !dg || !(eps >= 0.f)) return CYFA_ERR_ARG;
    if (!aligned16(o) || !aligned16(z) || !aligned16(dy) || !aligned16(d_o) || !aligned16(dz))
        return CYFA_ERR_ALIGN;
    const Shape s = shape_of(dims);
    if (!workspace || workspace_bytes < mixer_workspace(s)) return CYFA_ERR_WORKSPACE;
    return cuda_status(launch_mixer_post_bwd(s, o, z, g, eps, dy, d_o, dz, dg, workspace,
                                             static_cast<cudaStream_t>(stream)));
}

int cyfa_check(void* stream) {
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(st) != cudaSuccess) return CYFA_ERR_CUDA;
    int err = 0, err2 = 0, err3 = 0, err4 = 0, err5 = 0;
    if (tc_read_error(st, &err) != cudaSuccess) return CYFA_ERR_CUDA;
    if (tc_bwd_read_error(st, &err2) != cudaSuccess) return CYFA_ERR_CUDA;
    if (prep_read_error(st, &err3) != cudaSuccess) return CYFA_ERR_CUDA;
    if (simt_fwd_read_error(st, &err4) != cudaSuccess) return CYFA_ERR_CUDA;
    if (simt_bwd_read_error(st, &err5) != cudaSuccess) return CYFA_ERR_CUDA;
    // a timeout is reported first (its results are incomplete), then invalid sequence offsets
    // (every result after them is meaningless), then a range error (results inexact)
    if (err == CYFA_ERR_TIMEOUT || err2 == CYFA_ERR_TIMEOUT) return CYFA_ERR_TIMEOUT;
    if (err3 == CYFA_ERR_ARG) return CYFA_ERR_ARG;
    if (err == CYFA_ERR_RANGE || err2 == CYFA_ERR_RANGE) return CYFA_ERR_RANGE;
    // otherwise any error word: a CUDA-core chunk kernel launched outside its layout (err4, err5)
    return (err || err2 || err3 || err4 || err5) ? CYFA_ERR_CUDA : CYFA_OK;
}

}  // extern "C"
