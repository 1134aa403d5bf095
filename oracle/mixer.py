"""The CyFA mixer's neighbours of the operator, float64 -- test infrastructure only.

Sec. 3.4 (Mixer and backbone) names them without formulas; the readings taken here are:

* ShortConv: a causal depthwise convolution of width K (4) over tokens, one filter per channel,
  zero before the first token, followed by SiLU (the convention of the linear-RNN mixers the
  paper cites):  u_t[c] = sum_{i<K} w[c, i] x_{t-K+1+i}[c],  a_t[c] = u_t[c] sigmoid(u_t[c]).
* QK RMSNorm: per (token, head) over the head dimension, with a gain g shared by the heads:
  rms(a) = a / sqrt(mean(a^2) + eps) * g.  Applied to the convolved queries and keys; the values
  keep the convolution and SiLU only.
* Output: head-wise RMSNorm of the operator output o (gain g_o) times a sigmoid gate whose logits
  z (from the mixer's low-rank gate projection) are given:  y = rms(o) * sigmoid(z).

The projections (W x) are plain matrix products outside these functions.  Gradients are the
chain rule of the lines above, written out; tests/test_oracle_mixer.py pins every function
(identity and delay filters against the definition, np.convolve per channel, RMS of the output,
scale invariance, SiLU values) and every gradient by central finite differences.
"""
import numpy as np

from .gates import sigmoid


def short_conv(x, w):
    """x [N, T, C], w [C, K] -> u [N, T, C], causal, zero history."""
    N, T, C = x.shape
    K = w.shape[1]
    u = np.zeros((N, T, C))
    for i in range(K):
        lag = K - 1 - i                       # tap i reads token t - lag
        if lag >= T:
            continue
        u[:, lag:, :] += w[None, None, :, i] * x[:, :T - lag, :]
    return u


def silu(u):
    return u * sigmoid(u)


def silu_grad(u):
    s = sigmoid(u)
    return s * (1.0 + u * (1.0 - s))


def rms_norm(a, g, eps):
    """a [..., d] normalised over its last axis, times the gain g [d]."""
    r = 1.0 / np.sqrt(np.mean(a * a, axis=-1, keepdims=True) + eps)
    return a * r * g


def rms_norm_backward(a, g, eps, dy):
    """Gradients of sum(rms_norm(a, g, eps) * dy) with respect to a and g (summed over rows)."""
    d = a.shape[-1]
    r = 1.0 / np.sqrt(np.mean(a * a, axis=-1, keepdims=True) + eps)
    e = dy * g
    da = r * e - a * r ** 3 * np.sum(e * a, axis=-1, keepdims=True) / d
    dg = np.sum((dy * a * r).reshape(-1, d), axis=0)
    return da, dg


def mixer_pre(xq, xk, xv, wq, wk, wv, gq, gk, eps, H):
    """ShortConv + SiLU on q, k, v ([N, T, H*d] inputs, [H*d, K] filters), then RMSNorm per head
    on q and k.  Returns (q, k, v) as [N, T, H*d]."""
    N, T, C = xq.shape
    d = C // H
    aq, ak, av = (silu(short_conv(x, w)) for x, w in ((xq, wq), (xk, wk), (xv, wv)))
    q = rms_norm(aq.reshape(N, T, H, d), gq, eps).reshape(N, T, C)
    k = rms_norm(ak.reshape(N, T, H, d), gk, eps).reshape(N, T, C)
    return q, k, av


def conv_silu_backward(x, w, da):
    """Gradients of sum(silu(short_conv(x, w)) * da) with respect to x and w."""
    N, T, C = x.shape
    K = w.shape[1]
    u = short_conv(x, w)
    du = da * silu_grad(u)
    dx = np.zeros_like(x)
    dw = np.zeros_like(w)
    for i in range(K):
        lag = K - 1 - i
        if lag >= T:
            continue
        dx[:, :T - lag, :] += w[None, None, :, i] * du[:, lag:, :]
        dw[:, i] = np.sum(du[:, lag:, :] * x[:, :T - lag, :], axis=(0, 1))
    return dx, dw


def mixer_pre_backward(xq, xk, xv, wq, wk, wv, gq, gk, eps, H, dq, dk, dv):
    """Gradients of sum(q dq + k dk + v dv) for mixer_pre: (dxq, dxk, dxv, dwq, dwk, dwv, dgq, dgk)."""
    N, T, C = xq.shape
    d = C // H
    out = {}
    for name, x, w, g, dy in (('q', xq, wq, gq, dq), ('k', xk, wk, gk, dk)):
        a = silu(short_conv(x, w)).reshape(N, T, H, d)
        da, dg = rms_norm_backward(a, g, eps, dy.reshape(N, T, H, d))
        out['dx' + name], out['dw' + name] = conv_silu_backward(x, w, da.reshape(N, T, C))
        out['dg' + name] = dg
    out['dxv'], out['dwv'] = conv_silu_backward(xv, wv, dv)
    return out


def mixer_post(o, z, g, eps):
    """Head-wise RMSNorm of o [..., d] (gain g) times sigmoid(z)."""
    return rms_norm(o, g, eps) * sigmoid(z)


def mixer_post_backward(o, z, g, eps, dy):
    """Gradients of sum(mixer_post(o, z, g, eps) * dy): (do, dz, dg)."""
    s = sigmoid(z)
    n = rms_norm(o, g, eps)
    dz = dy * n * s * (1.0 - s)
    do, dg = rms_norm_backward(o, g, eps, dy * s)
    return do, dz, dg
