"""One drafting step of the hot path through the C ABI.

A step drafts every level of the draft chain/tree once: for each drafting
step d (Nq_d new nodes), the new nodes' q/k/v are RoPE'd and appended
(kvshot_draft_append), then the new nodes attend over [target prefix | draft
KV so far] (kvshot_draft_attn).  In "whole" mode all N nodes are appended
once and attend together (whole-tree verification shape).

Only device memory is handled here (torch allocations); all arithmetic runs
in libkvshot's kernels.
"""
from __future__ import annotations

from typing import List, Optional

import torch

from . import kvshot
from . import workloads as wl


class DraftStep:
    def __init__(self, inp: wl.Inputs, mode: str = "per_depth", flags: int = 0, num_ctas: int = 0,
                 scale: float = 0.0, err_flag: bool = True, target_fp8=None, qk_norm=None):
        """target_fp8: optional (codes_k, codes_v, k_scale_exp, v_scale_exp), an e4m3 copy of the target
        cache (workloads.fp8_target) to attend instead of inp.target_k / inp.target_v.
        qk_norm: optional (q_norm_w, k_norm_w, eps): the append normalises q and k per head first
        (kvshot_draft_append_qknorm)."""
        if mode not in ("per_depth", "whole"):
            raise ValueError(mode)
        self.inp, self.mode = inp, mode
        self.qk_norm = qk_norm
        s = inp.spec
        k_exp = v_exp = 0
        if target_fp8 is not None:
            self.target_k, self.target_v, k_exp, v_exp = target_fp8
            flags |= kvshot.KVSHOT_TARGET_FP8
        else:
            self.target_k, self.target_v = inp.target_k, inp.target_v
        dev = inp.target_k.device
        self.device = dev
        C, N = s.num_caches, s.n_nodes
        self.draft_k = torch.zeros((C, s.hkv, inp.n_max, s.head_dim), dtype=torch.bfloat16, device=dev)
        self.draft_v = torch.zeros_like(self.draft_k)
        self.err = torch.zeros(1, dtype=torch.int32, device=dev) if err_flag else None
        if mode == "per_depth":
            self.levels = list(s.levels)
            self.q_in, self.k_in, self.v_in, self.pos = inp.q_in, inp.k_in, inp.v_in, inp.positions
        else:
            self.levels = [N]
            self.q_in = [torch.cat(inp.q_in, dim=1)]
            self.k_in = [torch.cat(inp.k_in, dim=1)]
            self.v_in = [torch.cat(inp.v_in, dim=1)]
            self.pos = [torch.cat(inp.positions, dim=1).contiguous()]
        self.q_rot: List[torch.Tensor] = [torch.empty_like(q) for q in self.q_in]
        self.out: List[torch.Tensor] = [torch.empty_like(q) for q in self.q_in]
        self.lse: List[torch.Tensor] = [torch.empty(q.shape[:3], dtype=torch.float32, device=dev) for q in self.q_in]
        paged = inp.page_table is not None
        self.descs = []
        self.parents: List[torch.Tensor] = []  # [B, n_nodes] of each call (tree_parent's row stride is n_nodes)
        n0 = 0
        for n_step in self.levels:
            n0 += n_step
            self.parents.append(inp.tree_parent[:, :n0].contiguous())
            self.descs.append(kvshot.make_desc(
                num_caches=C, num_seqs=s.num_seqs, hq=s.hq, hkv=s.hkv, n_nodes=n0, n_query=n_step,
                n_max=inp.n_max, max_seq_len=s.max_seq_len, head_dim=s.head_dim,
                page_size=s.page_size if paged else 0,
                max_pages_per_seq=inp.page_table.shape[1] if paged else 0,
                num_pages=inp.num_pages if paged else 0, l_cap=inp.l_cap, scale=scale, tree=s.tree,
                # the attention call follows this step's own append kernel, which writes only q and the draft K/V
                flags=flags | kvshot.KVSHOT_OVERLAP_PREVIOUS, num_ctas=num_ctas, err_flag=self.err,
                k_scale_exp=k_exp, v_scale_exp=v_exp))
        ws = max(kvshot.workspace_size(d) for d in self.descs)
        if ws == 0:
            raise kvshot.KvshotError(kvshot.KVSHOT_ERR_SHAPE, "kvshot_draft_attn_workspace_size")
        self.workspace = torch.empty(ws, dtype=torch.uint8, device=dev)
        for d in self.descs:
            d.workspace = self.workspace.data_ptr()
            d.workspace_bytes = ws

    @property
    def tokens(self) -> int:
        """Draft tokens produced per step (a token attending several reused layers counts once)."""
        return self.inp.spec.num_seqs * self.inp.spec.n_nodes

    def run(self, stream: Optional[torch.cuda.Stream] = None) -> None:
        inp = self.inp
        n0 = 0
        for i, n_step in enumerate(self.levels):
            d = self.descs[i]
            if self.qk_norm is not None:
                wq, wk, eps = self.qk_norm
                kvshot.draft_append_qknorm(d, self.q_in[i], self.k_in[i], self.v_in[i], self.pos[i], n0, n_step,
                                           inp.spec.rope_base, wq, wk, eps, self.draft_k, self.draft_v,
                                           self.q_rot[i], stream)
            else:
                kvshot.draft_append(d, self.q_in[i], self.k_in[i], self.v_in[i], self.pos[i], n0, n_step,
                                    inp.spec.rope_base, self.draft_k, self.draft_v, self.q_rot[i], stream)
            kvshot.draft_attn(d, self.q_rot[i], self.target_k, self.target_v, inp.page_table, inp.seq_lens,
                              self.draft_k, self.draft_v, self.parents[i], self.out[i], self.lse[i], stream)
            n0 += n_step

    def error_code(self) -> int:
        return int(self.err.item()) if self.err is not None else 0
