"""Seeded synthetic inputs for the CyFA operator.

This module holds no part of the operator's arithmetic.  It draws the
inputs that both the CUDA library (through the tests and ``bench.py``) and the
fp64 oracle consume, with the shapes and value distributions of the paper's
400M-1.4B training layers:

* q, k ~ N(0, 1), each (token, head) vector L2-normalised along d (the mixer
  applies a norm to queries and keys before the operator, Sec. 3.4);
* v ~ N(0, 1);
* clock, decay and write-strength logits ~ N(0, 1), float32, [B, T, H];
* upstream gradient dO ~ N(0, 1);
* readout R_h = I + 0.02 N(0, 1) per head (the paper initialises R = I);
* decay scale A_h log-spaced over [1/256, 1]: A_h = 256^(-h/(H-1)).

Tensors are [B, T, H, d] row-major.  For bf16 runs q, k, v and dO are cast
to bfloat16 with round-to-nearest-even after drawing in float32; the oracle is
then fed those exact bf16 values widened to float64.
"""
import math

import torch

M_ACTIVE = 127      # active relative-time slots used by the paper's implementation
M_STORE = 128       # storage rows (one padding row)


def decay_scales(H):
    """A_h = 256^(-h/(H-1)) for h = 0..H-1 (A = 1 for a single head)."""
    if H == 1:
        return torch.ones(1, dtype=torch.float32)
    h = torch.arange(H, dtype=torch.float64)
    return torch.pow(256.0, -h / (H - 1)).to(torch.float32)


def readout_init(H, m=M_ACTIVE, seed=0, jitter=0.02, identity=False):
    """R [H, m, m] float32 = I + jitter * N(0,1) (exactly I with ``identity``)."""
    g = torch.Generator(device='cpu').manual_seed(seed + 7919)
    R = torch.eye(m, dtype=torch.float32).expand(H, m, m).clone()
    if not identity:
        R += jitter * torch.randn(H, m, m, generator=g, dtype=torch.float32)
    return R


def _unit(x):
    return x / torch.linalg.vector_norm(x, dim=-1, keepdim=True)


def make_inputs(B, T, H, d, *, seed=0, dtype=torch.bfloat16, device='cpu', with_dO=False,
                identity_R=False, m=M_ACTIVE):
    """Draw one workload.  Returns a dict of tensors on ``device``.

    Draw order: q, k, v, clock_logit, decay_logit, beta_logit, dO (if asked).
    R and A_h come from their own streams so they do not depend on T.
    """
    g = torch.Generator(device=device).manual_seed(seed)
    kw = dict(generator=g, device=device, dtype=torch.float32)
    q = _unit(torch.randn(B, T, H, d, **kw)).to(dtype)
    k = _unit(torch.randn(B, T, H, d, **kw)).to(dtype)
    v = torch.randn(B, T, H, d, **kw).to(dtype)
    clock = torch.randn(B, T, H, **kw)
    decay = torch.randn(B, T, H, **kw)
    beta = torch.randn(B, T, H, **kw)
    out = dict(q=q, k=k, v=v, clock_logit=clock, decay_logit=decay, beta_logit=beta)
    if with_dO:
        out['dO'] = torch.randn(B, T, H, d, **kw).to(dtype)
    out['R'] = readout_init(H, m=m, seed=seed, identity=identity_R).to(device)
    out['A'] = decay_scales(H).to(device)
    out['scale'] = 1.0 / math.sqrt(d)
    return out


def pair_view(x, b, h):
    """Slice one (batch, head) sequence out of a [B, T, H, ...] tensor as float64 numpy."""
    return x[b, :, h].detach().to('cpu', torch.float64).numpy()


def varlen_lengths(total, mean, *, seed=0, sigma=0.75, max_len=None):
    """Lengths of the sequences of one packed stream of `total` tokens: log-normal around `mean`
    (log-space spread sigma), each at least 1 and at most max_len, the last one taking what is
    left so that they sum to `total`.  A stand-in for a batch of documents of mixed length."""
    g = torch.Generator(device='cpu').manual_seed(seed + 104729)
    mu = math.log(mean) - 0.5 * sigma * sigma
    out, used = [], 0
    while used < total:
        x = math.exp(mu + sigma * float(torch.randn(1, generator=g)))
        n = max(1, int(round(x)))
        if max_len:
            n = min(n, max_len)
        n = min(n, total - used)
        out.append(n)
        used += n
    return out
