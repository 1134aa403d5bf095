"""Per-token gates and the cumulative clock, float64 -- test infrastructure only.

* delta_t = sigmoid(clock_logit_t) in (0,1)           Sec. 3.4 Eq. clock_gradient_stabilization
* lambda_t = lambda_{t-1} + delta_t, lambda_0 given   Sec. 3.1 Eq. cyfa-cumulative-clock
* alpha_t = exp(-A softplus(decay_logit_t))           Sec. 3.4 (scalar forget gate)
* beta_t  = sigmoid(beta_logit_t)                     Sec. 3.1 states only beta in (0,1);
  the sigmoid is this library's reading (the paper names no activation).

Pins (tests/test_oracle_gates.py): sigmoid(0) = 1/2, the symmetry sigmoid(x) +
sigmoid(-x) = 1, the exact rationals sigmoid(+-ln n) and the logistic definition at
sample points; softplus(0) = ln 2, softplus(x) - softplus(-x) = x, its limits and
its derivative (sigmoid); forget_gate(0, A) = 2^-A, its limits 1 and 0, its range
(0, 1] and monotonicity, and additivity in A; write_strength in (0, 1); lambda
against the closed form of a constant-rate clock and Prop. 5 (order preservation).
"""
import numpy as np


def sigmoid(x):
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * (1.0 + np.tanh(0.5 * x))


def softplus(x):
    x = np.asarray(x, dtype=np.float64)
    return np.logaddexp(0.0, x)


def clock_increment(clock_logit):
    return sigmoid(clock_logit)


def forget_gate(decay_logit, A):
    """alpha = exp(-A softplus(decay_logit)); A broadcasts against the logits."""
    return np.exp(-np.asarray(A, dtype=np.float64) * softplus(decay_logit))


def write_strength(beta_logit):
    return sigmoid(beta_logit)


def cumulative_clock(delta, lambda0=0.0, axis=-1):
    """lambda_t = lambda0 + sum_{u<=t} delta_u along ``axis`` (Eq. cyfa-cumulative-clock)."""
    lam = np.cumsum(np.asarray(delta, dtype=np.float64), axis=axis)
    return lam + lambda0
