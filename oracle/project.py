"""CPU fp64 oracle for the KV-only drafter's multi-layer KV projection -- numpy.

TEST INFRASTRUCTURE ONLY.  Only tests, the package's ``smoke()`` self-check and
``bench.py``'s CPU-baseline leg may import it; the library never does, and
nothing here imports the library.

Definition (arXiv 2604.26412, Sec. 3.2, injection strategy "linear
projection" and its "Proj + RoPE fix" variant).  For a verified token with
the K and V vectors K_l, V_l in R^{d_kv} (d_kv = hkv x 128, all KV heads) of
the L sampled target layers l = 1..L:

    K' = W_K [K_1; ...; K_L],   V' = W_V [V_1; ...; V_L],   W_K, W_V in R^{d_kv x L d_kv}

and, in the RoPE-fix variant, K' is rotated by RoPE at the token's position
(rotate-half pairs (j, j + 64) of every 128-wide head,
theta_j = pos * base^(-2j/128); the reading stated in the design notes).
The results are placed in the token's slot of the single reused cache.
Everything is fp64; bf16 inputs (uint16 bit patterns) are widened exactly.
"""
from __future__ import annotations

import numpy as np

from .fusion import widen

HEAD_DIM = 128


def rope(x: np.ndarray, pos: np.ndarray, base: float) -> np.ndarray:
    """Rotate every 128-wide head of x [T, hkv*128] by its token's position pos [T]."""
    T, dkv = x.shape
    h = x.reshape(T, dkv // HEAD_DIM, HEAD_DIM)
    j = np.arange(HEAD_DIM // 2, dtype=np.float64)
    theta = pos.astype(np.float64)[:, None] * base ** (-2.0 * j / HEAD_DIM)  # [T, 64]
    c, s = np.cos(theta)[:, None, :], np.sin(theta)[:, None, :]
    a, b = h[..., :HEAD_DIM // 2], h[..., HEAD_DIM // 2:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1).reshape(T, dkv)


def kv_project(k_in, v_in, w_k, w_v, positions, rope_base: float, apply_rope: bool):
    """K' and V' [T, d_kv] in fp64 for k_in, v_in [T, L, hkv, 128] and w_k, w_v [d_kv, L d_kv]."""
    k, v, wk, wv = (widen(x) for x in (k_in, v_in, w_k, w_v))
    T, L, hkv, D = k.shape
    if D != HEAD_DIM or v.shape != k.shape or wk.shape != (hkv * D, L * hkv * D) or wv.shape != wk.shape:
        raise ValueError("kv_project: inconsistent shapes")
    kp = k.reshape(T, L * hkv * D) @ wk.T  # [K_1; ...; K_L] per token
    vp = v.reshape(T, L * hkv * D) @ wv.T
    if apply_rope:
        kp = rope(kp, np.asarray(positions), rope_base)
    return kp, vp


def cache_rows(token_cache, positions, hkv: int, page_table=None, page_size: int = 0, l_cap: int = 0):
    """Row index [T, hkv] of each token's (cache, position) slot in a [rows, 128] view of the cache pool."""
    c = np.asarray(token_cache, dtype=np.int64)
    p = np.asarray(positions, dtype=np.int64)
    h = np.arange(hkv, dtype=np.int64)[None, :]
    if page_table is not None:
        pid = np.asarray(page_table, dtype=np.int64)[c, p // page_size]
        return (pid[:, None] * hkv + h) * page_size + (p % page_size)[:, None]
    return (c[:, None] * hkv + h) * l_cap + p[:, None]
