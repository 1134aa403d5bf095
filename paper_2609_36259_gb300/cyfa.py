"""Thin Python binding of libcyfa.so (include/cyfa.h): argument marshalling only.

Each function has the name of the C entry point it calls and takes torch tensors, passing
their device pointers and the current CUDA stream.  All arithmetic runs in the library's
kernels; when the library cannot be loaded the call raises (there is no fallback path).
"""
import ctypes
import os

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, 'libcyfa.so')

CYFA_OK = 0
CYFA_ERR_ARG, CYFA_ERR_SHAPE, CYFA_ERR_ALIGN, CYFA_ERR_WORKSPACE = -1, -2, -3, -4
CYFA_ERR_CUDA, CYFA_ERR_TIMEOUT, CYFA_ERR_UNSUPPORTED, CYFA_ERR_RANGE = -5, -6, -7, -8
CYFA_DTYPE_BF16, CYFA_DTYPE_FP32 = 0, 1
CYFA_WS_PREPARE, CYFA_WS_FWD, CYFA_WS_BWD, CYFA_WS_PREPARE_VARLEN, CYFA_WS_MIXER = 0, 1, 2, 3, 4

# Every symbol include/cyfa.h declares (checked by tests/test_abi.py).
EXPORTS = ('cyfa_version', 'cyfa_error_string', 'cyfa_workspace_size', 'cyfa_prepare',
           'cyfa_chunk_fwd', 'cyfa_chunk_bwd', 'cyfa_step', 'cyfa_check', 'cyfa_stats_reset',
           'cyfa_stats_timing', 'cyfa_stats_get', 'cyfa_prepare_noalloc',
           'cyfa_selftest_mma', 'cyfa_saved_size', 'cyfa_selftest_timeout',
           'cyfa_prepare_fixed_rate', 'cyfa_prepare_varlen', 'cyfa_mixer_pre',
           'cyfa_mixer_pre_bwd', 'cyfa_mixer_post', 'cyfa_mixer_post_bwd')


class CyfaError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__('%s (code %d)' % (msg, code))
        self.code = code


class Dims(ctypes.Structure):
    _fields_ = [('B', ctypes.c_int), ('T', ctypes.c_int), ('H', ctypes.c_int),
                ('dk', ctypes.c_int), ('dv', ctypes.c_int), ('m', ctypes.c_int),
                ('chunk', ctypes.c_int), ('scale', ctypes.c_float), ('dtype', ctypes.c_int),
                ('flags', ctypes.c_int)]


CYFA_FLAG_CUDA_CORES = 1


def storage_rows(m):
    """Rows of a state for m active slots: 128 for m <= 127, 256 above (rows m.. stay zero)."""
    return 128 if m <= 127 else 256


def dims(B, T, H, d, *, chunk=64, scale=None, dtype=torch.bfloat16, m=127, cuda_cores=False):
    return Dims(B, T, H, d, d, m, chunk, float(d ** -0.5 if scale is None else scale),
                CYFA_DTYPE_BF16 if dtype == torch.bfloat16 else CYFA_DTYPE_FP32,
                CYFA_FLAG_CUDA_CORES if cuda_cores else 0)


_lib = None
_VP = ctypes.c_void_p


def load(path=LIB_PATH):
    """Load libcyfa.so (once) and declare the C signatures."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError('libcyfa.so not built at %s: run __graft_entry__.build()' % path)
    lib = ctypes.CDLL(path)
    P = ctypes.POINTER(Dims)
    lib.cyfa_version.restype = ctypes.c_int
    lib.cyfa_error_string.restype = ctypes.c_char_p
    lib.cyfa_error_string.argtypes = [ctypes.c_int]
    lib.cyfa_workspace_size.argtypes = [P, ctypes.c_int, ctypes.POINTER(ctypes.c_size_t)]
    lib.cyfa_prepare.argtypes = [P] + [_VP] * 9 + [_VP, ctypes.c_size_t, _VP]
    lib.cyfa_saved_size.argtypes = [P, ctypes.POINTER(ctypes.c_size_t)]
    lib.cyfa_chunk_fwd.argtypes = [P] + [_VP] * 14 + [ctypes.c_size_t, _VP]
    lib.cyfa_chunk_bwd.argtypes = [P] + [_VP] * 21 + [ctypes.c_size_t, _VP]
    lib.cyfa_step.argtypes = [P] + [_VP] * 13
    lib.cyfa_check.argtypes = [_VP]
    lib.cyfa_selftest_mma.argtypes = [ctypes.c_int, _VP, _VP, _VP, _VP]
    lib.cyfa_selftest_timeout.argtypes = [ctypes.c_uint, _VP, _VP]
    lib.cyfa_prepare_noalloc.argtypes = [P] + [_VP] * 9 + [_VP]
    lib.cyfa_prepare_fixed_rate.argtypes = [P, ctypes.c_double] + [_VP] * 8 + [_VP]
    lib.cyfa_prepare_varlen.argtypes = ([P, _VP, ctypes.c_int, _VP, ctypes.c_double] + [_VP] * 8
                                        + [_VP, ctypes.c_size_t, _VP])
    F = ctypes.c_float
    lib.cyfa_mixer_pre.argtypes = [P] + [_VP] * 8 + [F] + [_VP] * 3 + [_VP]
    lib.cyfa_mixer_pre_bwd.argtypes = ([P] + [_VP] * 8 + [F] + [_VP] * 11 + [_VP, ctypes.c_size_t,
                                                                             _VP])
    lib.cyfa_mixer_post.argtypes = [P, _VP, _VP, _VP, F, _VP, _VP]
    lib.cyfa_mixer_post_bwd.argtypes = [P, _VP, _VP, _VP, F, _VP, _VP, _VP, _VP, _VP,
                                        ctypes.c_size_t, _VP]
    lib.cyfa_stats_timing.argtypes = [ctypes.c_int]
    lib.cyfa_stats_get.argtypes = [ctypes.c_int, ctypes.c_char_p, ctypes.c_int,
                                   ctypes.POINTER(ctypes.c_longlong), ctypes.POINTER(ctypes.c_double)]
    for name in EXPORTS:
        getattr(lib, name).restype = ctypes.c_int if name != 'cyfa_error_string' else ctypes.c_char_p
    _lib = lib
    return lib


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _ok(code):
    if code != CYFA_OK:
        raise CyfaError(code, load().cyfa_error_string(code).decode())


def error_string(code):
    return load().cyfa_error_string(code).decode()


def version():
    return load().cyfa_version()


def cyfa_workspace_size(d, which):
    n = ctypes.c_size_t(0)
    _ok(load().cyfa_workspace_size(ctypes.byref(d), which, ctypes.byref(n)))
    return n.value


def workspace(d, which, device='cuda'):
    return torch.empty(max(1, cyfa_workspace_size(d, which)), dtype=torch.uint8, device=device)


def cyfa_saved_size(d):
    n = ctypes.c_size_t(0)
    _ok(load().cyfa_saved_size(ctypes.byref(d), ctypes.byref(n)))
    return n.value


def saved_buffer(d, device='cuda'):
    """Buffer for the forward's saved chunk-start states (None where nothing is saved)."""
    n = cyfa_saved_size(d)
    return torch.empty(n, dtype=torch.uint8, device=device) if n else None


def cyfa_prepare(d, clock_logit, decay_logit, beta_logit, A, lambda0, lam_mod, g_cum, beta,
                 lambda_end, ws, stream=None):
    _ok(load().cyfa_prepare(ctypes.byref(d), _ptr(clock_logit), _ptr(decay_logit),
                            _ptr(beta_logit), _ptr(A), _ptr(lambda0), _ptr(lam_mod), _ptr(g_cum),
                            _ptr(beta), _ptr(lambda_end), _ptr(ws), ws.numel(), _stream(stream)))


def cyfa_prepare_noalloc(d, clock_logit, decay_logit, beta_logit, A, lambda0, lam_mod, g_cum,
                         beta, lambda_end, stream=None):
    """cyfa_prepare without a workspace, for callers that must not allocate device memory
    (its partial sums use a fixed array inside the library; see include/cyfa.h)."""
    _ok(load().cyfa_prepare_noalloc(ctypes.byref(d), _ptr(clock_logit), _ptr(decay_logit),
                                    _ptr(beta_logit), _ptr(A), _ptr(lambda0), _ptr(lam_mod),
                                    _ptr(g_cum), _ptr(beta), _ptr(lambda_end), _stream(stream)))


def cyfa_prepare_fixed_rate(d, rho, decay_logit, beta_logit, A, lambda0, lam_mod, g_cum, beta,
                            lambda_end, stream=None):
    _ok(load().cyfa_prepare_fixed_rate(ctypes.byref(d), float(rho), _ptr(decay_logit),
                                       _ptr(beta_logit), _ptr(A), _ptr(lambda0), _ptr(lam_mod),
                                       _ptr(g_cum), _ptr(beta), _ptr(lambda_end), _stream(stream)))


def cyfa_prepare_varlen(d, cu_seqlens, nseq, clock_logit, rho, decay_logit, beta_logit, A,
                        lambda0, lam_mod, g_cum, beta, lambda_end, ws, stream=None):
    _ok(load().cyfa_prepare_varlen(ctypes.byref(d), _ptr(cu_seqlens), int(nseq),
                                   _ptr(clock_logit), float(rho), _ptr(decay_logit),
                                   _ptr(beta_logit), _ptr(A), _ptr(lambda0), _ptr(lam_mod),
                                   _ptr(g_cum), _ptr(beta), _ptr(lambda_end), _ptr(ws),
                                   ws.numel(), _stream(stream)))


def cyfa_chunk_fwd(d, q, k, v, lam_mod, g_cum, beta, R, Kbar0, Vbar0, o, Kbar_out, Vbar_out, ws,
                   stream=None, saved=None):
    _ok(load().cyfa_chunk_fwd(ctypes.byref(d), _ptr(q), _ptr(k), _ptr(v), _ptr(lam_mod),
                              _ptr(g_cum), _ptr(beta), _ptr(R), _ptr(Kbar0), _ptr(Vbar0), _ptr(o),
                              _ptr(Kbar_out), _ptr(Vbar_out), _ptr(saved), _ptr(ws), ws.numel(),
                              _stream(stream)))


def cyfa_chunk_bwd(d, q, k, v, lam_mod, g_cum, beta, R, clock_logit, decay_logit, A, dO, dq, dk,
                   dv, d_clock_logit, d_decay_logit, d_beta_logit, dR, dA, ws, stream=None,
                   saved=None):
    _ok(load().cyfa_chunk_bwd(ctypes.byref(d), _ptr(q), _ptr(k), _ptr(v), _ptr(lam_mod),
                              _ptr(g_cum), _ptr(beta), _ptr(R), _ptr(clock_logit),
                              _ptr(decay_logit), _ptr(A), _ptr(dO), _ptr(dq), _ptr(dk), _ptr(dv),
                              _ptr(d_clock_logit), _ptr(d_decay_logit), _ptr(d_beta_logit),
                              _ptr(dR), _ptr(dA), _ptr(saved), _ptr(ws), ws.numel(),
                              _stream(stream)))


def cyfa_step(d, q, k, v, clock_logit, decay_logit, beta_logit, A, R, Kbar, Vbar, lam, o,
              stream=None):
    _ok(load().cyfa_step(ctypes.byref(d), _ptr(q), _ptr(k), _ptr(v), _ptr(clock_logit),
                         _ptr(decay_logit), _ptr(beta_logit), _ptr(A), _ptr(R), _ptr(Kbar),
                         _ptr(Vbar), _ptr(lam), _ptr(o), _stream(stream)))


def cyfa_mixer_pre(d, xq, xk, xv, wq, wk, wv, gq, gk, eps, q, k, v, stream=None):
    _ok(load().cyfa_mixer_pre(ctypes.byref(d), *map(_ptr, (xq, xk, xv, wq, wk, wv, gq, gk)),
                              float(eps), _ptr(q), _ptr(k), _ptr(v), _stream(stream)))


def cyfa_mixer_pre_bwd(d, xq, xk, xv, wq, wk, wv, gq, gk, eps, dq, dk, dv, dxq, dxk, dxv, dwq, dwk,
                       dwv, dgq, dgk, ws, stream=None):
    _ok(load().cyfa_mixer_pre_bwd(ctypes.byref(d), *map(_ptr, (xq, xk, xv, wq, wk, wv, gq, gk)),
                                  float(eps), *map(_ptr, (dq, dk, dv, dxq, dxk, dxv, dwq, dwk,
                                                          dwv, dgq, dgk)),
                                  _ptr(ws), ws.numel(), _stream(stream)))


def cyfa_mixer_post(d, o, z, g, eps, y, stream=None):
    _ok(load().cyfa_mixer_post(ctypes.byref(d), _ptr(o), _ptr(z), _ptr(g), float(eps), _ptr(y),
                               _stream(stream)))


def cyfa_mixer_post_bwd(d, o, z, g, eps, dy, d_o, dz, dg, ws, stream=None):
    _ok(load().cyfa_mixer_post_bwd(ctypes.byref(d), _ptr(o), _ptr(z), _ptr(g), float(eps),
                                   _ptr(dy), _ptr(d_o), _ptr(dz), _ptr(dg), _ptr(ws), ws.numel(),
                                   _stream(stream)))


def cyfa_check(stream=None):
    _ok(load().cyfa_check(_stream(stream)))


def cyfa_selftest_mma(variant, X, Y, D, stream=None):
    _ok(load().cyfa_selftest_mma(variant, _ptr(X), _ptr(Y), _ptr(D), _stream(stream)))


def cyfa_selftest_timeout(limit_us, elapsed_ns=None, stream=None):
    """Run the bounded-wait expiry self-check with a wait limit of limit_us microseconds;
    returns the library's status code (not raised: CYFA_ERR_TIMEOUT is the expected outcome)."""
    return load().cyfa_selftest_timeout(limit_us, _ptr(elapsed_ns), _stream(stream))


def cyfa_stats_reset():
    _ok(load().cyfa_stats_reset())


def cyfa_stats_timing(on):
    _ok(load().cyfa_stats_timing(1 if on else 0))


def cyfa_stats_get():
    """{kernel name: (launches, total ms)} for every kernel launched since the last reset."""
    lib = load()
    out = {}
    i = 0
    buf = ctypes.create_string_buffer(128)
    n = ctypes.c_longlong()
    ms = ctypes.c_double()
    while lib.cyfa_stats_get(i, buf, 128, ctypes.byref(n), ctypes.byref(ms)) == CYFA_OK:
        out[buf.value.decode()] = (n.value, ms.value)
        i += 1
    return out


# ---- convenience: whole calls with library-owned outputs (still argument marshalling) ----

def prepare(d, clock_logit, decay_logit, beta_logit, A, lambda0=None, want_lambda_end=False):
    B, T, H = clock_logit.shape
    dev = clock_logit.device
    lam = torch.empty(B, T, H, dtype=torch.float32, device=dev)
    g = torch.empty_like(lam)
    beta = torch.empty_like(lam)
    lend = torch.empty(B, H, dtype=torch.float64, device=dev) if want_lambda_end else None
    ws = workspace(d, CYFA_WS_PREPARE, dev)
    cyfa_prepare(d, clock_logit, decay_logit, beta_logit, A, lambda0, lam, g, beta, lend, ws)
    return lam, g, beta, lend


def prepare_varlen(d, cu_seqlens, decay_logit, beta_logit, A, clock_logit=None, rho=0.0,
                   lambda0=None, want_lambda_end=False):
    B, T, H = decay_logit.shape
    dev = decay_logit.device
    nseq = cu_seqlens.numel() - 1
    lam = torch.empty(B, T, H, dtype=torch.float32, device=dev)
    g = torch.empty_like(lam)
    beta = torch.empty_like(lam)
    lend = torch.empty(nseq, H, dtype=torch.float64, device=dev) if want_lambda_end else None
    ws = workspace(d, CYFA_WS_PREPARE_VARLEN, dev)
    cyfa_prepare_varlen(d, cu_seqlens, nseq, clock_logit, rho, decay_logit, beta_logit, A,
                        lambda0, lam, g, beta, lend, ws)
    return lam, g, beta, lend


def prepare_fixed_rate(d, rho, decay_logit, beta_logit, A, lambda0=None, want_lambda_end=False):
    B, T, H = decay_logit.shape
    dev = decay_logit.device
    lam = torch.empty(B, T, H, dtype=torch.float32, device=dev)
    g = torch.empty_like(lam)
    beta = torch.empty_like(lam)
    lend = torch.empty(B, H, dtype=torch.float64, device=dev) if want_lambda_end else None
    cyfa_prepare_fixed_rate(d, rho, decay_logit, beta_logit, A, lambda0, lam, g, beta, lend)
    return lam, g, beta, lend


def forward(d, q, k, v, lam, g, beta, R, Kbar0=None, Vbar0=None, want_state=False, ws=None,
            saved=None):
    o = torch.empty_like(v)
    B, T, H, D = v.shape
    Ko = Vo = None
    if want_state:
        Ko = torch.empty(B, H, storage_rows(d.m), D, dtype=torch.float32, device=v.device)
        Vo = torch.empty_like(Ko)
    if ws is None:
        ws = workspace(d, CYFA_WS_FWD, v.device)
    cyfa_chunk_fwd(d, q, k, v, lam, g, beta, R, Kbar0, Vbar0, o, Ko, Vo, ws, saved=saved)
    return o, Ko, Vo
