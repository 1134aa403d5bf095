"""torch.autograd wrappers of the library's calls and the CyFA mixer built from them (Sec. 3.4).

Every forward and backward here is a call of libcyfa.so through the C ABI (cyfa.py); PyTorch
supplies the parameters, the plain projections (matrix products) and the autograd graph.

* ``CyfaFunction``       -- the operator: cyfa_prepare + cyfa_chunk_fwd (keeping the chunk-start
                            states for the backward where the kernels save them) and
                            cyfa_chunk_bwd; gradients for q, k, v, the three logits, A and R.
* ``MixerPreFunction``   -- cyfa_mixer_pre / cyfa_mixer_pre_bwd (ShortConv + SiLU, QK RMSNorm).
* ``MixerPostFunction``  -- cyfa_mixer_post / cyfa_mixer_post_bwd (head RMSNorm, sigmoid gate).
* ``CyfaMixer``          -- projections, the three functions and the output projection, with the
                            clock stop-gradient of Eq. clock_gradient_stabilization: the clock
                            logits are projected from a detached copy of the layer input, so the
                            clock path trains W_delta and b_delta but sends no gradient into x.
"""
import math

import torch

from . import cyfa


def _dims(x, chunk, scale, m, cuda_cores=False):
    B, T, H, D = x.shape
    return cyfa.dims(B, T, H, D, chunk=chunk, scale=scale, dtype=x.dtype, m=m,
                     cuda_cores=cuda_cores)


class CyfaFunction(torch.autograd.Function):
    """o = CyFA(q, k, v; clock, decay, beta logits, A, R) for [B, T, H, d] inputs."""

    @staticmethod
    def forward(ctx, q, k, v, clock_logit, decay_logit, beta_logit, A, R, scale, chunk):
        q, k, v = (t.contiguous() for t in (q, k, v))
        logits = [t.contiguous().float() for t in (clock_logit, decay_logit, beta_logit)]
        m = R.shape[-1]
        d = _dims(q, chunk, scale, m)
        lam, g, beta, _ = cyfa.prepare(d, *logits, A.contiguous().float())
        saved = cyfa.saved_buffer(d, q.device)
        Rf = R.contiguous().float()
        o = cyfa.forward(d, q, k, v, lam, g, beta, Rf, saved=saved)[0]
        ctx.save_for_backward(q, k, v, *logits, A.contiguous().float(), Rf, lam, g, beta,
                              saved if saved is not None else torch.empty(0, device=q.device))
        ctx.d = d
        ctx.has_saved = saved is not None
        return o

    @staticmethod
    def backward(ctx, dO):
        q, k, v, c, f, bl, A, R, lam, g, beta, saved = ctx.saved_tensors
        d = ctx.d
        dO = dO.contiguous().to(q.dtype)
        dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
        dc, df, db = torch.empty_like(c), torch.empty_like(f), torch.empty_like(bl)
        dA, dR = torch.empty_like(A), torch.empty_like(R)
        ws = cyfa.workspace(d, cyfa.CYFA_WS_BWD, q.device)
        cyfa.cyfa_chunk_bwd(d, q, k, v, lam, g, beta, R, c, f, A, dO, dq, dk, dv, dc, df, db, dR,
                            dA, ws, saved=saved if ctx.has_saved else None)
        return dq, dk, dv, dc, df, db, dA, dR, None, None


class MixerPreFunction(torch.autograd.Function):
    """(q, k, v) = ShortConv + SiLU of the projections, RMSNorm on q and k."""

    @staticmethod
    def forward(ctx, xq, xk, xv, wq, wk, wv, gq, gk, eps, chunk):
        xs = [t.contiguous() for t in (xq, xk, xv)]
        ps = [t.contiguous().float() for t in (wq, wk, wv, gq, gk)]
        d = _dims(xs[0], chunk, 1.0, 127)
        out = [torch.empty_like(t) for t in xs]
        cyfa.cyfa_mixer_pre(d, *xs, *ps, eps, *out)
        ctx.save_for_backward(*xs, *ps)
        ctx.d, ctx.eps = d, eps
        return tuple(out)

    @staticmethod
    def backward(ctx, dq, dk, dv):
        xq, xk, xv, wq, wk, wv, gq, gk = ctx.saved_tensors
        dys = [t.contiguous().to(xq.dtype) for t in (dq, dk, dv)]
        dxs = [torch.empty_like(t) for t in (xq, xk, xv)]
        dws = [torch.empty_like(t) for t in (wq, wk, wv)]
        dgs = [torch.empty_like(t) for t in (gq, gk)]
        ws = cyfa.workspace(ctx.d, cyfa.CYFA_WS_MIXER, xq.device)
        cyfa.cyfa_mixer_pre_bwd(ctx.d, xq, xk, xv, wq, wk, wv, gq, gk, ctx.eps, *dys, *dxs, *dws,
                                *dgs, ws)
        return (*dxs, *dws, *dgs, None, None)


class MixerPostFunction(torch.autograd.Function):
    """y = RMSNorm(o) * g * sigmoid(z), per (token, head)."""

    @staticmethod
    def forward(ctx, o, z, g, eps, chunk):
        o, z = o.contiguous(), z.contiguous().to(o.dtype)
        g = g.contiguous().float()
        d = _dims(o, chunk, 1.0, 127)
        y = torch.empty_like(o)
        cyfa.cyfa_mixer_post(d, o, z, g, eps, y)
        ctx.save_for_backward(o, z, g)
        ctx.d, ctx.eps = d, eps
        return y

    @staticmethod
    def backward(ctx, dy):
        o, z, g = ctx.saved_tensors
        dy = dy.contiguous().to(o.dtype)
        d_o, dz, dg = torch.empty_like(o), torch.empty_like(z), torch.empty_like(g)
        ws = cyfa.workspace(ctx.d, cyfa.CYFA_WS_MIXER, o.device)
        cyfa.cyfa_mixer_post_bwd(ctx.d, o, z, g, ctx.eps, dy, d_o, dz, dg, ws)
        return d_o, dz, dg, None, None


class CyfaMixer(torch.nn.Module):
    """One CyFA mixer (Sec. 3.4): projections of x to q, k, v (ShortConv + SiLU, QK RMSNorm),
    the clock / decay / write-strength logits per head, the operator, head RMSNorm with a
    low-rank sigmoid output gate, and the output projection.  The clock logits see x.detach()
    (Eq. clock_gradient_stabilization).  Parameters in fp32; activations in `dtype`."""

    def __init__(self, d_model, H, d_head, m=127, gate_rank=16, chunk=64, eps=1e-6,
                 dtype=torch.bfloat16, device='cuda'):
        super().__init__()
        kw = dict(device=device, dtype=torch.float32)
        C = H * d_head
        self.H, self.d, self.m, self.chunk, self.eps, self.dtype = H, d_head, m, chunk, eps, dtype
        lin = torch.nn.Linear
        self.w_q, self.w_k, self.w_v = (lin(d_model, C, bias=False, **kw) for _ in range(3))
        self.w_clock, self.w_decay, self.w_beta = (lin(d_model, H, **kw) for _ in range(3))
        self.A_log = torch.nn.Parameter(torch.log(torch.linspace(1.0, 1.0 / 256, H, **kw)))
        self.R = torch.nn.Parameter(torch.eye(m, **kw).repeat(H, 1, 1))    # identity at start
        conv = torch.zeros(3, C, 4, **kw)
        conv[:, :, 3] = 1.0                       # the ShortConv starts as the identity
        self.conv = torch.nn.Parameter(conv)
        self.g_q, self.g_k, self.g_o = (torch.nn.Parameter(torch.ones(d_head, **kw))
                                        for _ in range(3))
        self.gate_down = lin(d_model, gate_rank, bias=False, **kw)
        self.gate_up = lin(gate_rank, C, **kw)
        self.w_out = lin(C, d_model, bias=False, **kw)

    def forward(self, x):
        B, T, _ = x.shape
        H, d = self.H, self.d
        dt = self.dtype

        def heads(t):
            return t.to(dt).reshape(B, T, H, d)
        xq, xk, xv = heads(self.w_q(x)), heads(self.w_k(x)), heads(self.w_v(x))
        q, k, v = MixerPreFunction.apply(xq, xk, xv, self.conv[0], self.conv[1], self.conv[2],
                                         self.g_q, self.g_k, self.eps, self.chunk)
        clock = self.w_clock(x.detach())         # stop-gradient into x on the clock path
        o = CyfaFunction.apply(q, k, v, clock, self.w_decay(x), self.w_beta(x),
                               torch.exp(self.A_log), self.R, 1.0 / math.sqrt(d), self.chunk)
        z = heads(self.gate_up(self.gate_down(x)))
        y = MixerPostFunction.apply(o, z, self.g_o, self.eps, self.chunk)
        return self.w_out(y.reshape(B, T, H * d).float())
