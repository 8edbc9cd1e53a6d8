"""Seeded synthetic inputs for the draft-attention hot path.

This module only *generates inputs*: tensor shapes, seeded random values,
page tables, draft-tree parent arrays and RoPE positions.  It holds none of
the attention arithmetic, so both the CUDA library's tests/benchmarks and the
CPU oracle's checks can draw from it.

The shapes stand in for the paper's Qwen3-8B runs (target model Qwen3-8B,
Sec. 3.1; GQA 32 query / 8 KV heads, head dim 128).  The paper's ShareGPT /
UltraChat data and trained weights are not used: keys/values are N(0, 1)
(post-RoPE target K is just a bf16 tensor to the drafter), queries are
N(0, 1)/sqrt(128), as a drafter projection of unit-variance hidden states
would give.  Draft trees follow tree verification (Sec. 3.5, tree
(8, 10, 60)): level-by-level, every node's parent is drawn uniformly from the
previous level, with a fan-out cap.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional

import numpy as np
import torch

HQ, HKV, HEAD_DIM = 32, 8, 128
ROPE_BASE = 1.0e6  # Qwen3 rotary base


@dataclasses.dataclass
class Spec:
    """One draft-attention workload (a row of the benchmark configuration list)."""

    name: str
    num_seqs: int                 # B
    layers: int                   # reused target layers attended separately (caches per sequence)
    seq_lens: List[int]           # verified prefix length per cache, len == B * layers
    levels: List[int]             # draft nodes added per drafting step (chain: [1] * depth)
    tree: bool
    paged: bool
    page_size: int = 16
    hq: int = HQ
    hkv: int = HKV
    head_dim: int = HEAD_DIM
    max_fanout: int = 8
    seed: int = 0
    rope_base: float = ROPE_BASE

    @property
    def num_caches(self) -> int:
        return self.num_seqs * self.layers

    @property
    def n_nodes(self) -> int:
        return int(sum(self.levels))

    @property
    def max_seq_len(self) -> int:
        return int(max(self.seq_lens)) if self.seq_lens else 0


def config(idx: int, seed: int = 0) -> Spec:
    """The five benchmark workloads (1-based index), seeded."""
    rng = np.random.default_rng(seed + 1000 * idx)
    if idx == 1:   # tiny chain: B=1, L=128, contiguous, chain depth 4
        return Spec("tiny-chain-L128-d4", 1, 1, [128], [1] * 4, False, False, seed=seed)
    if idx == 2:   # KV-only chain: B=1, L=2048, contiguous, chain depth 8
        return Spec("kvonly-chain-L2048-d8", 1, 1, [2048], [1] * 8, False, False, seed=seed)
    if idx == 3:   # hybrid tree: B=16, L=4096, paged P=16, 64-node tree of depth 6
        return Spec("hybrid-tree-B16-L4096-n64-P16", 16, 1, [4096] * 16, [8, 12, 12, 12, 12, 8], True, True,
                    page_size=16, seed=seed)
    if idx == 4:   # ragged serving: B=64, L ~ U[512, 8192], paged P=16 shuffled, chain depth 8
        lens = rng.integers(512, 8192, size=64, endpoint=True).tolist()
        return Spec("ragged-chain-B64-L512to8192-d8-P16", 64, 1, lens, [1] * 8, False, True, page_size=16,
                    seed=seed)
    if idx == 5:   # long-context multi-layer: B=4 x 4 layers, L=32768, paged P=64, 32-node tree depth 8
        return Spec("multilayer-tree-B4x4-L32768-n32-P64", 4, 4, [32768] * 16, [4] * 8, True, True,
                    page_size=64, seed=seed)
    raise ValueError(f"no workload {idx}")


def tree_parents(levels: List[int], tree: bool, rng: np.random.Generator, max_fanout: int = 8) -> np.ndarray:
    """Parent array of one sequence's draft nodes, nodes numbered level by level.

    Level-1 nodes hang off the last verified token (parent -1).  A chain has
    parent[i] = i - 1.  In a tree each node draws its parent uniformly from the
    previous level, redrawing while that parent already has max_fanout children.
    """
    n = int(sum(levels))
    parent = np.full(n, -1, np.int32)
    if not tree:
        parent[1:] = np.arange(n - 1, dtype=np.int32)
        return parent
    start_prev, start = 0, 0
    for li, size in enumerate(levels):
        if li > 0:
            prev = np.arange(start_prev, start)
            kids = {int(p): 0 for p in prev}
            for i in range(start, start + size):
                while True:
                    p = int(rng.choice(prev))
                    if kids[p] < max_fanout:
                        break
                kids[p] += 1
                parent[i] = p
        start_prev, start = start, start + size
    return parent


def node_depths(levels: List[int]) -> np.ndarray:
    """1-based drafting step of each node (level index + 1)."""
    return np.concatenate([np.full(s, i + 1, np.int32) for i, s in enumerate(levels)]) if levels else \
        np.zeros(0, np.int32)


def rope_positions(seq_lens: List[int], levels: List[int], n0: int, n_new: int) -> np.ndarray:
    """RoPE positions [C, n_new] of nodes n0 .. n0+n_new-1: prefix length + depth - 1.

    Depth-1 nodes sit right after the last verified token (position L_c), and
    all nodes of one drafting step share a position (tree-attention convention).
    """
    dep = node_depths(levels)[n0:n0 + n_new]
    lens = np.asarray(seq_lens, np.int64)[:, None]
    return (lens + dep[None, :] - 1).astype(np.int32)


@dataclasses.dataclass
class Inputs:
    """Device-resident tensors for one workload (bf16 unless stated)."""

    spec: Spec
    seq_lens: torch.Tensor          # int32 [C]
    target_k: torch.Tensor          # paged [num_pages, hkv, P, D]  /  contiguous [C, hkv, l_cap, D]
    target_v: torch.Tensor
    page_table: Optional[torch.Tensor]  # int32 [C, max_pages] or None
    num_pages: int
    l_cap: int
    tree_parent: torch.Tensor       # int32 [B, N]
    n_max: int
    q_in: List[torch.Tensor]        # per step: [C, n_step, hq, D]
    k_in: List[torch.Tensor]        # per step: [C, n_step, hkv, D]
    v_in: List[torch.Tensor]
    positions: List[torch.Tensor]   # per step: int32 [C, n_step]


def _randn_bf16(shape, gen, device, std=1.0):
    return (torch.randn(shape, generator=gen, device=device, dtype=torch.float32) * std).to(torch.bfloat16)


def make_inputs(spec: Spec, device="cpu", seed: Optional[int] = None, tail_fill: str = "random") -> Inputs:
    """Generate a workload's tensors with a seeded torch.Generator on `device`.

    tail_fill: contents of cache rows past each sequence's prefix length
    (inside the last page / the contiguous capacity): "random" or "nan".
    """
    seed = spec.seed if seed is None else seed
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    rng = np.random.default_rng(seed)
    C, B, D = spec.num_caches, spec.num_seqs, spec.head_dim
    lens = np.asarray(spec.seq_lens, np.int64)
    assert len(lens) == C
    if spec.paged:
        P = spec.page_size
        pages_per = [(int(L) + P - 1) // P for L in lens]
        num_pages = int(sum(pages_per))
        max_pages = max(1, max(pages_per) if pages_per else 1)
        perm = rng.permutation(num_pages).astype(np.int32)
        table = np.zeros((C, max_pages), np.int32)
        cur = 0
        for c in range(C):
            table[c, :pages_per[c]] = perm[cur:cur + pages_per[c]]
            cur += pages_per[c]
        page_table = torch.from_numpy(table).to(device)
        shape = (max(num_pages, 1), spec.hkv, P, D)
        l_cap = 0
    else:
        num_pages = 0
        l_cap = int(max(int(lens.max()) if C else 0, 1))
        page_table = None
        shape = (C, spec.hkv, l_cap, D)
    target_k = _randn_bf16(shape, gen, device)
    target_v = _randn_bf16(shape, gen, device)
    if tail_fill == "nan":
        _fill_tails(spec, target_k, target_v, page_table, lens, float("nan"))
    N = spec.n_nodes
    n_max = max(8, ((N + 7) // 8) * 8)
    parents = np.stack([tree_parents(spec.levels, spec.tree, rng, spec.max_fanout) for _ in range(B)]) \
        if N else np.zeros((B, 0), np.int32)
    q_in, k_in, v_in, pos = [], [], [], []
    n0 = 0
    for n_step in spec.levels:
        q_in.append(_randn_bf16((C, n_step, spec.hq, D), gen, device, 1.0 / math.sqrt(D)))
        k_in.append(_randn_bf16((C, n_step, spec.hkv, D), gen, device))
        v_in.append(_randn_bf16((C, n_step, spec.hkv, D), gen, device))
        pos.append(torch.from_numpy(rope_positions(spec.seq_lens, spec.levels, n0, n_step)).to(device))
        n0 += n_step
    return Inputs(spec, torch.from_numpy(lens.astype(np.int32)).to(device), target_k, target_v, page_table,
                  num_pages, l_cap, torch.from_numpy(parents.astype(np.int32)).to(device), n_max,
                  q_in, k_in, v_in, pos)


def _fill_tails(spec, tk, tv, page_table, lens, value):
    if spec.paged:
        P = spec.page_size
        for c, L in enumerate(lens):
            if L % P:
                page = int(page_table[c, int(L) // P])
                tk[page, :, int(L) % P:, :] = value
                tv[page, :, int(L) % P:, :] = value
    else:
        for c, L in enumerate(lens):
            tk[c, :, int(L):, :] = value
            tv[c, :, int(L):, :] = value


# Scale exponents of the fp8 target-cache variant: keys and values are cached as e4m3 codes of
# x / 2^exp, so that N(0, 1) entries use the middle of e4m3's range (|x| 2^3 stays far below 448).
FP8_K_EXP = -3
FP8_V_EXP = -2


def fp8_target(inp: Inputs, k_exp: int = FP8_K_EXP, v_exp: int = FP8_V_EXP):
    """e4m3 codes (uint8 tensors shaped like target_k) of target_k / 2^k_exp and target_v / 2^v_exp,
    rounded to nearest by torch's float8_e4m3fn conversion (NaN entries stay NaN codes).  This is
    how a target model would fill an fp8 cache; the library only reads the codes."""
    def enc(x, e):
        return (x.float() * 2.0 ** (-e)).to(torch.float8_e4m3fn).view(torch.uint8).contiguous()
    return enc(inp.target_k, k_exp), enc(inp.target_v, v_exp)


def draft_buffers(spec: Spec, n_max: int, device="cpu", fill: float = float("nan")):
    """Empty draft K/V buffers [C, hkv, n_max, D] pre-filled with `fill` (NaN by default,
    so reading an unwritten slot is caught)."""
    shape = (spec.num_caches, spec.hkv, n_max, spec.head_dim)
    return (torch.full(shape, fill, dtype=torch.bfloat16, device=device),
            torch.full(shape, fill, dtype=torch.bfloat16, device=device))


def random_draft_kv(spec: Spec, n_max: int, n_fill: int, device="cpu", seed: int = 1, tail=float("nan")):
    """Draft K/V buffers whose first n_fill slots hold N(0,1) values (the rest `tail`)."""
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    dk, dv = draft_buffers(spec, n_max, device, tail)
    if n_fill:
        shape = (spec.num_caches, spec.hkv, n_fill, spec.head_dim)
        dk[:, :, :n_fill] = _randn_bf16(shape, gen, device)
        dv[:, :, :n_fill] = _randn_bf16(shape, gen, device)
    return dk, dv


def random_queries(spec: Spec, n_query: int, device="cpu", seed: int = 2):
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    return _randn_bf16((spec.num_caches, n_query, spec.hq, spec.head_dim), gen, device,
                       1.0 / math.sqrt(spec.head_dim))


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> numpy uint16 bit patterns (host copy)."""
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def bits_to_bf16(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)


HIDDEN = HQ * HEAD_DIM  # d of the hybrid drafter (Qwen3-8B hidden size; the two branches' width)


@dataclasses.dataclass
class FusionInputs:
    """Inputs of the gated-delta fusion: the branches n, o [T, d] and the fusion weights (bf16)."""
    n: torch.Tensor
    o: torch.Tensor
    w_g: torch.Tensor       # [d, 3d]
    b_g: torch.Tensor       # [d]
    w_delta: torch.Tensor   # [d, d]


def fusion_inputs(T: int, d: int = HIDDEN, device="cpu", seed: int = 5) -> FusionInputs:
    """Seeded stand-ins for the hybrid drafter's fusion step (Sec. 3.4): the two attention branches
    ~N(0, 1) (attention outputs of unit-variance values), W_g ~N(0, 1/(3d)) and W_delta ~N(0, 1/d)
    so the gate's pre-activation and the projected correction stay O(1), b_g ~N(0, 0.1^2).  No trained
    weights exist here; these only fix shapes and scales."""
    g = torch.Generator().manual_seed(seed)
    t = dict(n=_randn_bf16((T, d), g, "cpu"), o=_randn_bf16((T, d), g, "cpu"),
             w_g=_randn_bf16((d, 3 * d), g, "cpu", std=1.0 / math.sqrt(3 * d)),
             b_g=_randn_bf16((d,), g, "cpu", std=0.1),
             w_delta=_randn_bf16((d, d), g, "cpu", std=1.0 / math.sqrt(d)))
    return FusionInputs(**{k: v.to(device) for k, v in t.items()})


@dataclasses.dataclass
class ProjectInputs:
    """Inputs of the multi-layer KV projection: the new tokens' K/V of L layers and W_K, W_V (bf16)."""
    k_in: torch.Tensor   # [T, L, hkv, 128]
    v_in: torch.Tensor
    w_k: torch.Tensor    # [hkv*128, L*hkv*128]
    w_v: torch.Tensor


def project_inputs(T: int, L: int = 3, hkv: int = HKV, device="cpu", seed: int = 7) -> ProjectInputs:
    """Seeded stand-ins for the KV-only drafter's projection (Sec. 3.2): K/V ~N(0, 1) like the target
    cache, W ~N(0, 1/(L d_kv)) so the projected vectors stay O(1).  L = 3 sampled layers (App. B)."""
    g = torch.Generator().manual_seed(seed)
    dkv = hkv * HEAD_DIM
    t = dict(k_in=_randn_bf16((T, L, hkv, HEAD_DIM), g, "cpu"), v_in=_randn_bf16((T, L, hkv, HEAD_DIM), g, "cpu"),
             w_k=_randn_bf16((dkv, L * dkv), g, "cpu", std=1.0 / math.sqrt(L * dkv)),
             w_v=_randn_bf16((dkv, L * dkv), g, "cpu", std=1.0 / math.sqrt(L * dkv)))
    return ProjectInputs(**{k: v.to(device) for k, v in t.items()})
