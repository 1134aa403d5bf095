"""The C ABI library builds, loads without a GPU, exports every symbol include/cyfa.h declares,
and rejects bad arguments on the host before anything is launched."""
import ctypes
import os
import re

import pytest
import torch

from paper_2609_36259_gb300 import cyfa

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope='module')
def lib():
    if not os.path.exists(cyfa.LIB_PATH):
        from paper_2609_36259_gb300 import build_lib
        build_lib.build()
    return cyfa.load()


def declared_symbols():
    text = open(os.path.join(ROOT, 'include', 'cyfa.h')).read()
    text = re.sub(r'/\*.*?\*/', '', text, flags=re.S)
    return sorted(set(re.findall(r'\b(cyfa_[a-z_]+)\s*\(', text)))


def test_exports_every_declared_symbol(lib):
    names = declared_symbols()
    assert set(names) == set(cyfa.EXPORTS), names
    for n in names:
        assert hasattr(lib, n), n


def test_version_and_errors(lib):
    assert cyfa.version() >= 100
    for code in (0, -1, -2, -3, -4, -5, -6, -7, -99):
        assert isinstance(cyfa.error_string(code), str)


def test_workspace_sizes(lib):
    d = cyfa.dims(2, 32768, 16, 128, chunk=128, cuda_cores=True)
    fwd = cyfa.cyfa_workspace_size(d, cyfa.CYFA_WS_FWD)
    # CUDA-core path: readout matrices (2 x H x 128 x 128 fp32) plus one [128 x 2D] fp32 state
    # per chunk
    assert fwd >= 2 * 16 * 128 * 128 * 4 + 2 * 16 * 256 * 128 * 256 * 4
    # tensor-core path: one fp32 [128 x 256] state per (b, h, 1024-token segment)
    d = cyfa.dims(2, 32768, 16, 128, chunk=128)
    fwd_tc = cyfa.cyfa_workspace_size(d, cyfa.CYFA_WS_FWD)
    assert 2 * 16 * 32 * 128 * 256 * 4 <= fwd_tc < fwd
    assert cyfa.cyfa_workspace_size(d, cyfa.CYFA_WS_BWD) > 0
    assert cyfa.cyfa_workspace_size(d, cyfa.CYFA_WS_PREPARE) >= 2 * 16 * 32 * 8
    # m = 255: 256 storage rows on the CUDA-core kernels, 64-token chunks forward and 32-token
    # chunks backward (readout matrices 2 x H x 256 x 256; one [256 x 2D] state per chunk)
    d = cyfa.dims(1, 2048, 4, 256, m=255)
    fwd255 = cyfa.cyfa_workspace_size(d, cyfa.CYFA_WS_FWD)
    assert fwd255 >= 2 * 4 * 256 * 256 * 4 + 4 * 32 * 256 * 512 * 4
    bwd255 = cyfa.cyfa_workspace_size(d, cyfa.CYFA_WS_BWD)
    assert bwd255 >= 2 * 4 * 64 * 256 * 512 * 4 + 2 * 4 * 2048 * 256 * 4


@pytest.mark.parametrize('field,value,code', [
    ('m', 64, cyfa.CYFA_ERR_SHAPE), ('m', 256, cyfa.CYFA_ERR_SHAPE), ('m', 0, cyfa.CYFA_ERR_SHAPE),
    ('m', 257, cyfa.CYFA_ERR_SHAPE), ('dk', 96, cyfa.CYFA_ERR_SHAPE),
    ('chunk', 32, cyfa.CYFA_ERR_SHAPE), ('T', 100, cyfa.CYFA_ERR_SHAPE), ('B', 0, cyfa.CYFA_ERR_ARG),
    ('dtype', 7, cyfa.CYFA_ERR_ARG), ('B', 65536, cyfa.CYFA_ERR_SHAPE)])
def test_bad_dims_rejected_on_host(lib, field, value, code):
    d = cyfa.dims(1, 128, 1, 128)
    setattr(d, field, value)
    n = ctypes.c_size_t()
    assert lib.cyfa_workspace_size(ctypes.byref(d), cyfa.CYFA_WS_FWD, ctypes.byref(n)) == code


def test_null_and_misaligned_pointers_rejected_on_host(lib):
    d = cyfa.dims(1, 128, 1, 128)
    nul = [None] * 14
    assert lib.cyfa_chunk_fwd(ctypes.byref(d), *nul, 0, None) == cyfa.CYFA_ERR_ARG
    bad = ctypes.c_void_p(0x1002)      # never dereferenced: rejected before any launch
    good = ctypes.c_void_p(0x1000)
    args = [bad, good, good, good, good, good, good, None, None, good, None, None, None, good]
    assert lib.cyfa_chunk_fwd(ctypes.byref(d), *args, 1 << 30, None) == cyfa.CYFA_ERR_ALIGN
    args = [good] * 7 + [None, None, good, None, None, bad, good]   # misaligned saved buffer
    assert lib.cyfa_chunk_fwd(ctypes.byref(d), *args, 1 << 30, None) == cyfa.CYFA_ERR_ALIGN
    args = [good] * 7 + [None, None, good, None, None, None, good]
    assert lib.cyfa_chunk_fwd(ctypes.byref(d), *args, 16, None) == cyfa.CYFA_ERR_WORKSPACE
    assert lib.cyfa_step(ctypes.byref(d), *([None] * 13)) == cyfa.CYFA_ERR_ARG


def test_saved_size(lib):
    """The saved chunk-start states: fp16 [B*H][T/128][2][128][128] and M [H][128][128] on the
    tensor-core path; fp32 [B*H][T/64][128][2d] on the CUDA-core kernels where their forward
    walks 64-token chunks with 128 storage rows (the backward's chunks); nothing otherwise."""
    B, T, H = 2, 1024, 3
    full = B * H * (T // 128) * 2 * 128 * 128 * 2 + H * 128 * 128 * 2   # states, then M
    simt = lambda d: B * H * (T // 64) * 128 * 2 * d * 4
    assert cyfa.cyfa_saved_size(cyfa.dims(B, T, H, 128)) == full
    assert cyfa.cyfa_saved_size(cyfa.dims(B, T, H, 128, m=63)) == full   # odd m in 63..127
    assert cyfa.cyfa_saved_size(cyfa.dims(B, T, H, 128, m=31)) == simt(128)
    assert cyfa.cyfa_saved_size(cyfa.dims(B, T, H, 128, m=255)) == 0   # 256 storage rows
    assert cyfa.cyfa_saved_size(cyfa.dims(B, T, H, 256)) == simt(256)
    assert cyfa.cyfa_saved_size(cyfa.dims(B, T, H, 256, chunk=128)) == simt(256)   # walks 64
    assert cyfa.cyfa_saved_size(cyfa.dims(B, T, H, 128, cuda_cores=True)) == simt(128)
    assert cyfa.cyfa_saved_size(cyfa.dims(B, T, H, 128, chunk=128, cuda_cores=True)) == 0
    assert cyfa.cyfa_saved_size(cyfa.dims(B, T, H, 64)) == simt(64)
    assert cyfa.cyfa_saved_size(cyfa.dims(B, T, H, 128, dtype=torch.float32)) == simt(128)


def test_timeout_selftest_rejects_bad_limits_on_host(lib):
    """The failure-detection self-check refuses a wait limit outside 1 us .. 1 s before any CUDA
    call (its GPU behaviour is tested in test_gpu_failure_detection.py)."""
    for limit in (0, 1000001, 2 ** 32 - 1):
        assert lib.cyfa_selftest_timeout(limit, None, None) == cyfa.CYFA_ERR_ARG


@pytest.mark.parametrize('field,value,code', [
    ('dtype', 7, cyfa.CYFA_ERR_ARG), ('m', 64, cyfa.CYFA_ERR_SHAPE), ('T', 100, cyfa.CYFA_ERR_SHAPE),
    ('B', 65536, cyfa.CYFA_ERR_SHAPE)])
def test_noalloc_prepare_checks_dims_like_prepare(lib, field, value, code):
    """cyfa_prepare_noalloc applies cyfa_prepare's argument checks, before any CUDA call."""
    d = cyfa.dims(1, 128, 1, 128)
    setattr(d, field, value)
    good = ctypes.c_void_p(0x1000)      # never dereferenced: rejected before any launch
    args = [good] * 4 + [None] + [good] * 3 + [None, None]
    assert lib.cyfa_prepare_noalloc(ctypes.byref(d), *args) == code
    assert lib.cyfa_prepare(ctypes.byref(d), *args[:9], good, 1 << 30, None) == code


def test_fixed_rate_and_varlen_prepare_check_arguments_on_host(lib):
    """Host-side refusals of cyfa_prepare_fixed_rate and cyfa_prepare_varlen (nothing launched)."""
    good = ctypes.c_void_p(0x1000)      # never dereferenced: rejected before any launch
    d = cyfa.dims(1, 128, 1, 128)
    for rho in (0.0, -1.0, float('nan')):
        assert lib.cyfa_prepare_fixed_rate(ctypes.byref(d), rho, *([good] * 3), None,
                                           *([good] * 3), None, None) == cyfa.CYFA_ERR_ARG
    n = ctypes.c_size_t()
    assert lib.cyfa_workspace_size(ctypes.byref(d), cyfa.CYFA_WS_PREPARE_VARLEN,
                                   ctypes.byref(n)) == 0 and n.value > 0

    def varlen(dd, nseq=2, clock=good, rho=0.0, ws_bytes=1 << 20):
        return lib.cyfa_prepare_varlen(ctypes.byref(dd), good, nseq, clock, rho, good, good, good,
                                       None, good, good, good, None, good, ws_bytes, None)
    assert varlen(cyfa.dims(2, 128, 1, 128)) == cyfa.CYFA_ERR_ARG          # B must be 1
    assert varlen(d, nseq=0) == cyfa.CYFA_ERR_ARG
    assert varlen(d, clock=None, rho=0.0) == cyfa.CYFA_ERR_ARG              # no clock, no rate
    assert varlen(d, ws_bytes=8) == cyfa.CYFA_ERR_WORKSPACE
    assert varlen(cyfa.dims(1, 100, 1, 128)) == cyfa.CYFA_ERR_SHAPE


def test_backward_clock_gradient_both_or_neither(lib):
    """cyfa_chunk_bwd takes no clock logits only together with no clock gradient."""
    good = ctypes.c_void_p(0x1000)
    d = cyfa.dims(1, 128, 1, 128)
    args = [good] * 21
    args[7] = None      # clock_logit missing, d_clock_logit given
    assert lib.cyfa_chunk_bwd(ctypes.byref(d), *args, 1 << 30, None) == cyfa.CYFA_ERR_ARG
    args = [good] * 21
    args[14] = None     # d_clock_logit missing, clock_logit given
    assert lib.cyfa_chunk_bwd(ctypes.byref(d), *args, 1 << 30, None) == cyfa.CYFA_ERR_ARG
