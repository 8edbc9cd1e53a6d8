"""CPU fp64 oracle for the hybrid drafter's gated-delta fusion -- numpy.

TEST INFRASTRUCTURE ONLY.  Only tests, the package's ``smoke()`` self-check and
``bench.py``'s CPU-baseline leg may import it; the library never does, and
nothing here imports the library.

Definition (arXiv 2604.26412, Sec. 3.4).  For a draft token with
self-attention branch output n (the EAGLE-3 path, Eq. "self-attn") and
cross-attention branch output o (re-attention to the target KV, Eq.
"cross-attn"), both in R^d:

    delta = o - n                                   (Eq. "delta")
    g     = sigmoid(W_g [n; o; delta] + b_g)        (Eq. "fusion")
    h     = n + g (.) (W_delta delta)               (Eq. "fusion")

with W_g in R^{d x 3d} and b_g in R^d shared across draft steps, W_delta in
R^{d x d}, sigmoid the logistic function and (.) the element-wise product.
Rows of the [T, d] arrays are tokens.  The computation follows the equations
in that order, in fp64, with numpy's matrix product as the only library step;
bf16 inputs (uint16 bit patterns) are widened exactly.
"""
from __future__ import annotations

import numpy as np


def widen(a) -> np.ndarray:
    """fp64 view of an array: uint16 arrays are taken as bf16 bit patterns, others are cast."""
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def sigmoid(z: np.ndarray) -> np.ndarray:
    """Logistic function 1 / (1 + e^-z), evaluated without overflow for either sign of z."""
    ez = np.exp(-np.abs(z))
    return np.where(z >= 0, 1.0 / (1.0 + ez), ez / (1.0 + ez))


def gated_delta(n, o, w_g, b_g, w_delta) -> np.ndarray:
    """h for every token: n, o [T, d]; w_g [d, 3d]; b_g [d]; w_delta [d, d].  Returns fp64 [T, d]."""
    n, o, w_g, b_g, w_delta = (widen(x) for x in (n, o, w_g, b_g, w_delta))
    T, d = n.shape
    if o.shape != (T, d) or w_g.shape != (d, 3 * d) or b_g.shape != (d,) or w_delta.shape != (d, d):
        raise ValueError("gated_delta: inconsistent shapes")
    delta = o - n
    x = np.concatenate([n, o, delta], axis=1)  # [n; o; delta] per token
    g = sigmoid(x @ w_g.T + b_g)
    return n + g * (delta @ w_delta.T)
