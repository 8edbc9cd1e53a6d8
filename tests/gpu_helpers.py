"""Helpers for the GPU parity tests: run the CPU oracle on (a subset of) a
device workload and compare the library's outputs with it.

Tolerances (bf16 inputs, fp32 accumulation, bf16 output):
  out: max |gpu - oracle| <= 2e-2 and ||gpu - oracle||_2 / ||oracle||_2 <= 5e-3
  lse: max |gpu - oracle| <= 1e-3 (natural log, fp32)
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import oracle
from paper_2604_26412_gb300 import workloads as wl

OUT_MAX_ABS = 2e-2
OUT_REL_L2 = 5e-3
LSE_MAX_ABS = 1e-3


class HostCache:
    """Host copies (uint16 bits) of a workload's target cache, made once."""

    def __init__(self, inp: wl.Inputs):
        self.inp = inp
        self.tk = wl.bf16_bits(inp.target_k)
        self.tv = wl.bf16_bits(inp.target_v)
        self.page_table = inp.page_table.cpu().numpy() if inp.page_table is not None else None
        self.seq_lens = inp.seq_lens.cpu().numpy()
        self.parents = inp.tree_parent.cpu().numpy()


def oracle_attn(hc: HostCache, q, draft_k, draft_v, n_nodes, n_query, caches=None, scale=0.0, tree=None,
                parents=None, seq_lens=None):
    """Oracle out/lse (float64) for the given caches (default: all)."""
    s = hc.inp.spec
    C = s.num_caches
    caches = list(range(C)) if caches is None else list(caches)
    per_seq = C // s.num_seqs
    qh = wl.bf16_bits(q)[caches]
    dk = wl.bf16_bits(draft_k)[caches]
    dv = wl.bf16_bits(draft_v)[caches]
    lens = (hc.seq_lens if seq_lens is None else np.asarray(seq_lens))[caches].astype(np.int32)
    par_all = hc.parents if parents is None else parents
    par = np.stack([par_all[c // per_seq][:n_nodes] for c in caches]).astype(np.int32)
    tree = s.tree if tree is None else tree
    n = len(caches)
    if hc.page_table is not None:
        d = oracle.make_desc(num_caches=n, num_seqs=n, hq=s.hq, hkv=s.hkv, head_dim=s.head_dim, n_nodes=n_nodes,
                             n_query=n_query, n_max=dk.shape[2], tree=tree, paged=True, page_size=s.page_size,
                             max_pages_per_seq=hc.page_table.shape[1], num_pages=hc.inp.num_pages, scale=scale)
        return oracle.attn(d, qh, hc.tk, hc.tv, hc.page_table[caches], lens, dk, dv, par)
    d = oracle.make_desc(num_caches=n, num_seqs=n, hq=s.hq, hkv=s.hkv, head_dim=s.head_dim, n_nodes=n_nodes,
                         n_query=n_query, n_max=dk.shape[2], tree=tree, l_cap=hc.inp.l_cap, scale=scale)
    return oracle.attn(d, qh, np.ascontiguousarray(hc.tk[caches]), np.ascontiguousarray(hc.tv[caches]), None, lens,
                       dk, dv, par)


def round_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp64 to the nearest bf16 (ties to even), as uint16 bit patterns, in exact integer arithmetic."""
    m, e = np.frexp(x)                      # x = m 2^e, 0.5 <= |m| < 1
    q = np.ldexp(m, 8)                       # 8 significant bits: |q| in [128, 256)
    r = np.rint(q)                           # numpy rounds half to even
    y = np.ldexp(r, e - 8).astype(np.float32)  # exact: at most 8 significant bits
    return (y.view(np.uint32) >> 16).astype(np.uint16)


def widen_bits(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns to fp64, exactly."""
    return (np.asarray(bits).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def compare(out_gpu: torch.Tensor, lse_gpu: torch.Tensor, out_ref: np.ndarray, lse_ref: np.ndarray, what=""):
    """Assert the tolerances; returns (max_abs, rel_l2, lse_err)."""
    o = out_gpu.float().cpu().numpy().astype(np.float64)
    l = lse_gpu.float().cpu().numpy().astype(np.float64)
    assert o.shape == out_ref.shape, (o.shape, out_ref.shape)
    assert np.all(np.isfinite(o)), f"{what}: non-finite output"
    diff = np.abs(o - out_ref)
    max_abs = float(diff.max()) if diff.size else 0.0
    rel = float(np.linalg.norm(o - out_ref) / max(np.linalg.norm(out_ref), 1e-30)) if diff.size else 0.0
    lse_err = float(np.abs(l - lse_ref).max()) if l.size else 0.0
    assert max_abs <= OUT_MAX_ABS, f"{what}: out max-abs {max_abs}"
    assert rel <= OUT_REL_L2, f"{what}: out rel-L2 {rel}"
    assert lse_err <= LSE_MAX_ABS, f"{what}: lse max-abs {lse_err}"
    return max_abs, rel, lse_err
