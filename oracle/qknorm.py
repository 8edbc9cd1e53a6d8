"""CPU fp64 oracle for the draft append with QK-norm -- numpy.

TEST INFRASTRUCTURE ONLY.  Only tests, the package's ``smoke()`` self-check and
``bench.py``'s CPU-baseline leg may import it; the library never does, and
nothing here imports the library.

Definition (arXiv 2604.26412, App. D "Additional Ablations", Tab. ablations,
the "QK-Norm" training regime; the paper names the variant only, so its form
is read from Qwen3's attention, which the drafter shares).  Before RoPE,
every 128-wide query and key head x is scaled to unit root-mean-square and by
a learned weight per dimension,

    RMSNorm(x) = x / sqrt(mean_j x_j^2 + eps) * w,

one weight vector w_q for all query heads and one w_k for all key heads; the
normalised heads are then rotated by RoPE at the node's position exactly as
in the plain append (rotate-half pairs (j, j + 64), theta_j = pos *
base^(-2j/128)).  Values are stored unchanged.  The rotated keys and values
go to draft slot n0 + i of their cache; the rotated queries are returned.
Everything is fp64; bf16 inputs (uint16 bit patterns) are widened exactly.
"""
from __future__ import annotations

import numpy as np

from .fusion import widen
from .project import rope

HEAD_DIM = 128


def rms_norm(x: np.ndarray, w: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm over the last axis (one head's 128 dims) of x, times the weights w [128]."""
    x = np.asarray(x, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)
    if x.shape[-1] != HEAD_DIM or w.shape != (HEAD_DIM,):
        raise ValueError("rms_norm: heads must be 128 wide")
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * w


def append_qknorm(q_in, k_in, v_in, positions, n0: int, rope_base: float, q_norm_w, k_norm_w, eps: float,
                  n_max: int):
    """q_in [C, n, hq, 128], k_in, v_in [C, n, hkv, 128] (bf16 bits), positions [C, n].

    Returns (q_out [C, n, hq, 128], k_slots [C, hkv, n, 128], v_slots [C, hkv, n, 128]) in fp64: the
    rotated queries and the contents of draft slots n0 .. n0 + n - 1.
    """
    q, k, v = widen(q_in), widen(k_in), widen(v_in)
    wq, wk = widen(q_norm_w), widen(k_norm_w)
    C, n, hq, D = q.shape
    hkv = k.shape[2]
    pos = np.asarray(positions, dtype=np.int64)
    if D != HEAD_DIM or k.shape != (C, n, hkv, D) or v.shape != k.shape or pos.shape != (C, n):
        raise ValueError("append_qknorm: inconsistent shapes")
    if not (eps > 0) or n0 < 0 or n0 + n > n_max:
        raise ValueError("append_qknorm: eps must be positive and the slots inside the draft region")
    flat_pos = pos.reshape(C * n)
    qn = rope(rms_norm(q, wq, eps).reshape(C * n, hq * D), flat_pos, rope_base).reshape(C, n, hq, D)
    kn = rope(rms_norm(k, wk, eps).reshape(C * n, hkv * D), flat_pos, rope_base).reshape(C, n, hkv, D)
    return qn, kn.transpose(0, 2, 1, 3), v.transpose(0, 2, 1, 3).copy()
