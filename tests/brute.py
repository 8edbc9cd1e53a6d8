"""Independent numpy fp64 brute force, used only to pin the CPU oracle.

It is written differently from the oracle on purpose: it gathers the whole
key matrix [prefix | all draft slots] per cache, builds an explicit 0/1 mask
from the transitive closure of the parent relation (matrix powers, not a
parent walk), evaluates the full score matrix with one matmul and takes
scipy's softmax over the masked row.
"""
from __future__ import annotations

import numpy as np
from scipy.special import softmax


def bits_to_f64(a: np.ndarray) -> np.ndarray:
    return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def reach_matrix(parent: np.ndarray) -> np.ndarray:
    """R[n, m] = 1 iff m == n or m is an ancestor of n (closure of the parent edge)."""
    n = len(parent)
    A = np.zeros((n, n), np.int64)
    for i, p in enumerate(parent):
        if p >= 0:
            A[i, p] = 1
    R = np.eye(n, dtype=np.int64)
    P = np.eye(n, dtype=np.int64)
    for _ in range(n):
        P = (P @ A > 0).astype(np.int64)
        R = R | P
    return R.astype(bool)


def gather_prefix(tk, page_table, c, h, L, paged, page_size):
    if paged:
        rows = [tk[page_table[c, j // page_size], h, j % page_size] for j in range(L)]
        return np.stack(rows) if rows else np.zeros((0, tk.shape[-1]), tk.dtype)
    return tk[c, h, :L]


def brute_attn(q, tk, tv, page_table, seq_lens, dk, dv, tree_parent, *, num_seqs, hq, hkv, n_nodes, n_query,
               tree, paged, page_size=0, scale=0.0):
    """q [C,Nq,hq,D], tk/tv cache arrays, dk/dv [C,hkv,n_max,D] (uint16 bits) -> out, lse (fp64)."""
    C, Nq, _, D = q.shape
    G = hq // hkv
    scale = scale if scale != 0.0 else 1.0 / np.sqrt(D)
    qf = bits_to_f64(q)
    out = np.zeros((C, Nq, hq, D))
    lse = np.zeros((C, Nq, hq))
    for c in range(C):
        seq = c // (C // num_seqs)
        parent = tree_parent[seq] if tree else np.arange(-1, n_nodes - 1)
        R = reach_matrix(np.asarray(parent))
        L = int(seq_lens[c])
        for h in range(hkv):
            K = np.concatenate([bits_to_f64(gather_prefix(tk, page_table, c, h, L, paged, page_size)),
                                bits_to_f64(dk[c, h, :n_nodes])])
            V = np.concatenate([bits_to_f64(gather_prefix(tv, page_table, c, h, L, paged, page_size)),
                                bits_to_f64(dv[c, h, :n_nodes])])
            for g in range(G):
                hh = h * G + g
                S = scale * (qf[c, :, hh, :] @ K.T)           # [Nq, L + N]
                mask = np.zeros_like(S, dtype=bool)
                mask[:, :L] = True
                for nl in range(Nq):
                    mask[nl, L:] = R[n_nodes - Nq + nl]
                S = np.where(mask, S, -np.inf)
                Pm = softmax(S, axis=1)
                out[c, :, hh, :] = Pm @ V
                mx = S.max(axis=1)
                lse[c, :, hh] = mx + np.log(np.exp(S - mx[:, None]).sum(axis=1))
    return out, lse
