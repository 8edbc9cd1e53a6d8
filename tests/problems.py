"""Small seeded problems for the tests (host numpy views of workloads.make_inputs)."""
from __future__ import annotations

import dataclasses

import numpy as np
import torch

from paper_2604_26412_gb300 import workloads as wl


@dataclasses.dataclass
class HostProblem:
    spec: wl.Spec
    q: np.ndarray            # uint16 [C, Nq, hq, D]
    tk: np.ndarray
    tv: np.ndarray
    page_table: np.ndarray   # int32 [C, max_pages] (zeros [C,1] when contiguous)
    seq_lens: np.ndarray     # int32 [C]
    dk: np.ndarray           # uint16 [C, hkv, n_max, D]
    dv: np.ndarray
    tree_parent: np.ndarray  # int32 [B, N]
    n_nodes: int
    n_query: int
    n_max: int
    num_pages: int
    l_cap: int

    def desc_kwargs(self, scale=0.0):
        s = self.spec
        return dict(num_caches=s.num_caches, num_seqs=s.num_seqs, hq=s.hq, hkv=s.hkv, head_dim=s.head_dim,
                    n_nodes=self.n_nodes, n_query=self.n_query, n_max=self.n_max, tree=s.tree, paged=s.paged,
                    page_size=s.page_size if s.paged else 0, max_pages_per_seq=self.page_table.shape[1],
                    num_pages=self.num_pages, l_cap=self.l_cap, scale=scale)

    def brute_kwargs(self, scale=0.0):
        s = self.spec
        return dict(num_seqs=s.num_seqs, hq=s.hq, hkv=s.hkv, n_nodes=self.n_nodes, n_query=self.n_query,
                    tree=s.tree, paged=s.paged, page_size=s.page_size, scale=scale)


def make(spec: wl.Spec, n_query=None, seed=0, n_nodes=None) -> HostProblem:
    """Host problem with draft slots 0..N-1 filled and queries for the last Nq nodes."""
    inp = wl.make_inputs(spec, "cpu", seed=seed)
    N = spec.n_nodes if n_nodes is None else n_nodes
    Nq = N if n_query is None else n_query
    n_max = inp.n_max
    dk, dv = wl.random_draft_kv(spec, n_max, N, "cpu", seed=seed + 11, tail=float("nan"))
    q = wl.random_queries(spec, Nq, "cpu", seed=seed + 22)
    pt = inp.page_table.numpy() if inp.page_table is not None else np.zeros((spec.num_caches, 1), np.int32)
    return HostProblem(spec, wl.bf16_bits(q), wl.bf16_bits(inp.target_k), wl.bf16_bits(inp.target_v), pt,
                       inp.seq_lens.numpy(), wl.bf16_bits(dk), wl.bf16_bits(dv), inp.tree_parent.numpy()[:, :N]
                       if N else inp.tree_parent.numpy(), N, Nq, n_max, inp.num_pages, inp.l_cap)


def small_spec(*, B=1, layers=1, lens=(20,), levels=(1, 1, 1), tree=False, paged=False, page_size=8, hq=4, hkv=2,
               D=8, seed=0, max_fanout=8):
    return wl.Spec("small", B, layers, list(lens), list(levels), tree, paged, page_size=page_size, hq=hq, hkv=hkv,
                   head_dim=D, seed=seed, max_fanout=max_fanout)
