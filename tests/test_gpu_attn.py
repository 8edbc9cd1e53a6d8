"""GPU parity of kvshot_draft_attn against the CPU fp64 oracle (through the C ABI).

Shapes span several 64-key tiles with ragged tails, empty prefixes, both cache
layouts and several page sizes, chains and trees, GQA groups 1/4/8/16/32, the
CUDA-core and tensor-core kernels (tensor-memory rows dense or spread),
single-row and multi-row-block stacks, and persistent grids from 1 CTA up (which changes how units are split into
pieces and merged).  Unused cache rows and draft slots hold NaN.
"""
import math

import numpy as np
import pytest
import torch

from paper_2604_26412_gb300 import kvshot
from paper_2604_26412_gb300 import workloads as wl
from tests import gpu_helpers as gh

pytestmark = pytest.mark.gpu


def _case(lens, levels, tree, paged, page_size=16, hq=32, hkv=8, n_query=None, seed=0, B=None, layers=1):
    B = B if B is not None else len(lens) // layers
    spec = wl.Spec("t", B, layers, list(lens), list(levels), tree, paged, page_size=page_size, hq=hq, hkv=hkv,
                   seed=seed)
    inp = wl.make_inputs(spec, "cuda", seed=seed, tail_fill="nan")
    N = spec.n_nodes
    Nq = N if n_query is None else n_query
    dk, dv = wl.random_draft_kv(spec, inp.n_max, N, "cuda", seed=seed + 1, tail=float("nan"))
    q = wl.random_queries(spec, Nq, "cuda", seed=seed + 2)
    return spec, inp, dk, dv, q, N, Nq


def _run(spec, inp, dk, dv, q, N, Nq, flags=0, num_ctas=0, scale=0.0, parents=None, ws=None):
    paged = inp.page_table is not None
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = kvshot.make_desc(num_caches=spec.num_caches, num_seqs=spec.num_seqs, hq=spec.hq, hkv=spec.hkv, n_nodes=N,
                         n_query=Nq, n_max=inp.n_max, max_seq_len=spec.max_seq_len,
                         page_size=spec.page_size if paged else 0,
                         max_pages_per_seq=inp.page_table.shape[1] if paged else 0,
                         num_pages=inp.num_pages if paged else 0, l_cap=inp.l_cap, scale=scale, tree=spec.tree,
                         flags=flags, num_ctas=num_ctas, err_flag=err)
    ws_bytes = kvshot.workspace_size(d)
    assert ws_bytes > 0
    if ws is None:
        ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    assert ws.numel() >= ws_bytes
    d.workspace, d.workspace_bytes = ws.data_ptr(), ws.numel()
    par = (inp.tree_parent[:, :N].contiguous() if parents is None else parents)
    kvshot.draft_attn(d, q, inp.target_k, inp.target_v, inp.page_table, inp.seq_lens, dk, dv, par, out, lse)
    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"device error {int(err.item())}"
    return out, lse


CASES = [
    # lens, levels, tree, paged, page_size, hq, hkv, n_query
    ((128,), (1, 1, 1, 1), False, False, 16, 32, 8, 1),          # tiny chain, one step
    ((200,), (1,) * 5, False, False, 16, 32, 8, 5),               # whole chain (20 rows -> mma)
    ((0,), (1, 1, 1), False, False, 16, 32, 8, 1),                # empty prefix
    ((1, 63, 64, 65), (1, 1), False, True, 16, 32, 8, 1),         # ragged around the tile size
    ((17, 130, 300), (4, 4), True, True, 8, 32, 8, 4),            # tree, 16 rows, P=8
    ((4096, 1000), (8, 12, 12), True, True, 16, 32, 8, 12),       # tree level of 12 nodes -> 48 rows
    ((257, 513), (8, 12, 12), True, True, 64, 32, 8, 32),         # 32 nodes -> 128 rows, 2 row blocks
    ((700,), (2, 3, 3), True, True, 128, 32, 8, 8),               # page larger than a tile
    ((333, 5), (3, 3), True, False, 16, 8, 8, 3),                 # G = 1
    ((90, 91, 92), (2, 2, 2), False, True, 16, 64, 8, 2),         # G = 8, chain of 6 nodes, 16 rows
    ((1500,), tuple([1] * 40), False, True, 16, 32, 8, 1),        # long chain: two draft tiles? (N = 40)
    ((65,), tuple([1] * 70), False, False, 16, 4, 4, 2),          # chain with N = 70 > one draft tile
    ((600, 129), (8, 12), True, True, 16, 32, 8, 20),             # 80 rows: dense TMEM rows, partial quarter
    ((300,), (2, 2), True, False, 16, 32, 2, 3),                  # G = 16: 48 rows spread, boxes of one node
    ((250, 70), (1, 1, 1), False, True, 16, 32, 1, 2),            # G = 32: 64 rows spread, boxes of 16 heads
    ((257, 513, 0), (8, 12, 12, 12), True, True, 16, 32, 8, 40),  # 160 rows: paired blocks, block 1 mostly empty
    ((1, 64, 130), (8, 12, 12, 12, 12, 8), True, True, 16, 32, 8, 64),  # 256 rows paired, ragged prefixes
    ((203,), tuple([1] * 40), False, False, 16, 32, 8, 40),       # whole chain: paired, contiguous l_cap % 8 != 0
    ((96, 200), tuple([1] * 100), False, True, 16, 32, 8, 100),   # 400 rows: two paired units per KV head
    ((500,), (4, 8, 8), True, True, 64, 64, 8, 20),               # G = 8: 160 rows paired, 64-token pages
    ((450, 31, 97), (2, 2), True, True, 32, 32, 8, 2),            # 32-token pages, ragged last page
    ((700, 65), (1, 1, 1), False, True, 192, 32, 8, 1),           # 192-token pages: 64-token slices of a page
]


@pytest.mark.parametrize("case", CASES, ids=[f"c{i}" for i in range(len(CASES))])
def test_attn_matches_oracle(case):
    lens, levels, tree, paged, P, hq, hkv, nq = case
    spec, inp, dk, dv, q, N, Nq = _case(lens, levels, tree, paged, P, hq, hkv, nq, seed=len(lens) + N_SEED(case))
    hc = gh.HostCache(inp)
    ref_out, ref_lse = gh.oracle_attn(hc, q, dk, dv, N, Nq)
    kernels = [0, kvshot.KVSHOT_FORCE_MMA] + ([kvshot.KVSHOT_FORCE_TC] if 128 % (hq // hkv) == 0 else [])
    for flags in kernels:
        for num_ctas in (0, 1, 7):
            out, lse = _run(spec, inp, dk, dv, q, N, Nq, flags=flags, num_ctas=num_ctas)
            gh.compare(out, lse, ref_out, ref_lse, f"{case} flags={flags} ctas={num_ctas}")


def N_SEED(case):
    return sum(case[1]) * 7 + (3 if case[2] else 0)


@pytest.mark.parametrize("flags", [kvshot.KVSHOT_FORCE_CC, kvshot.KVSHOT_FORCE_MMA, kvshot.KVSHOT_FORCE_TC])
@pytest.mark.parametrize("nq", [1, 3, 8])
def test_forced_kernels_agree_with_oracle(flags, nq):
    spec, inp, dk, dv, q, N, Nq = _case((300, 77), (2, 3, 3), True, True, 16, 32, 8, nq, seed=11)
    hc = gh.HostCache(inp)
    ref_out, ref_lse = gh.oracle_attn(hc, q, dk, dv, N, Nq)
    for num_ctas in (0, 3):
        out, lse = _run(spec, inp, dk, dv, q, N, Nq, flags=flags, num_ctas=num_ctas)
        gh.compare(out, lse, ref_out, ref_lse, f"flags={flags} nq={nq}")


def test_scale_parameter():
    spec, inp, dk, dv, q, N, Nq = _case((150,), (2, 2), True, True, 16, 32, 8, 2, seed=5)
    hc = gh.HostCache(inp)
    for scale in (1.0, 0.05):
        ref_out, ref_lse = gh.oracle_attn(hc, q, dk, dv, N, Nq, scale=scale)
        out, lse = _run(spec, inp, dk, dv, q, N, Nq, scale=scale)
        gh.compare(out, lse, ref_out, ref_lse, f"scale={scale}")


def test_deterministic_across_runs():
    spec, inp, dk, dv, q, N, Nq = _case((2000, 3000), (4, 4), True, True, 16, 32, 8, 4, seed=3)
    a = _run(spec, inp, dk, dv, q, N, Nq)
    b = _run(spec, inp, dk, dv, q, N, Nq)
    assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])


@pytest.mark.parametrize("flags", [0, kvshot.KVSHOT_FORCE_MMA, kvshot.KVSHOT_FORCE_TC])
@pytest.mark.parametrize("paged", [False, True])
@pytest.mark.parametrize("tree", [False, True])
def test_mask_probe_is_exact(paged, tree, flags):
    """q = 0 and one-hot V: every visible draft slot contributes exactly 1/n_vis to its own bucket."""
    lens = (37, 64, 129, 0) if paged else (37, 64, 129, 5)
    levels = (3, 5, 8, 8, 4) if tree else (1,) * 12
    spec, inp, dk, dv, q, N, Nq = _case(lens, levels, tree, paged, 16, 32, 8, None, seed=21)
    q.zero_()
    # prefix token j -> bucket j % 64 ; draft slot m -> bucket 64 + m
    D = 128
    inp.target_v.zero_()
    for c, L in enumerate(lens):
        for j in range(L):
            if paged:
                page = int(inp.page_table[c, j // 16])
                inp.target_v[page, :, j % 16, j % 64] = 1.0
            else:
                inp.target_v[c, :, j, j % 64] = 1.0
    dv[:, :, :N].zero_()
    for m in range(N):
        dv[:, :, m, 64 + m] = 1.0
    out, lse = _run(spec, inp, dk, dv, q, N, Nq, flags=flags)
    parents = inp.tree_parent.cpu().numpy()
    o = out.float().cpu().numpy()
    l = lse.cpu().numpy()
    for c, L in enumerate(lens):
        par = parents[c]
        for nl in range(Nq):
            n = N - Nq + nl
            vis = np.zeros(N, bool)
            m = n
            while m >= 0:
                vis[m] = True
                m = par[m] if tree else m - 1
            nvis = L + vis.sum()
            assert np.allclose(l[c, nl], math.log(nvis), atol=1e-5)
            got = np.rint(o[c, nl, :, 64:64 + N] * nvis).astype(int)
            assert np.array_equal(got, np.broadcast_to(vis.astype(int), got.shape)), (c, nl)


def test_device_errors_are_reported_without_fault():
    spec, inp, dk, dv, q, N, Nq = _case((100, 50), (2, 2), True, True, 16, 32, 8, 2, seed=9)
    # page id outside the pool
    saved = inp.page_table.clone()
    inp.page_table[1, 0] = inp.num_pages + 5
    with pytest.raises(AssertionError, match="device error 8"):
        _run(spec, inp, dk, dv, q, N, Nq)
    inp.page_table.copy_(saved)
    # sequence length above max_seq_len
    inp.seq_lens[0] = 10_000
    with pytest.raises(AssertionError, match="device error 8"):
        _run(spec, inp, dk, dv, q, N, Nq)
    inp.seq_lens[0] = 100
    # a parent that is not an earlier node
    par = inp.tree_parent[:, :N].clone()
    par[0, 3] = 3
    with pytest.raises(AssertionError, match="device error 5"):
        _run(spec, inp, dk, dv, q, N, Nq, parents=par)
    # and a clean call afterwards still works
    hc = gh.HostCache(inp)
    ref_out, ref_lse = gh.oracle_attn(hc, q, dk, dv, N, Nq)
    out, lse = _run(spec, inp, dk, dv, q, N, Nq)
    gh.compare(out, lse, ref_out, ref_lse, "after errors")


def test_workspace_too_small_is_rejected():
    spec, inp, dk, dv, q, N, Nq = _case((100,), (2,), True, True, 16, 32, 8, 2, seed=2)
    d = kvshot.make_desc(num_caches=1, num_seqs=1, hq=32, hkv=8, n_nodes=N, n_query=Nq, n_max=inp.n_max,
                         max_seq_len=100, page_size=16, max_pages_per_seq=inp.page_table.shape[1],
                         num_pages=inp.num_pages, tree=True)
    need = kvshot.workspace_size(d)
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    d.workspace, d.workspace_bytes = ws.data_ptr(), need - 1
    out = torch.empty_like(q)
    lse = torch.empty(q.shape[:3], dtype=torch.float32, device="cuda")
    st = kvshot.draft_attn_status(d, q, inp.target_k, inp.target_v, inp.page_table, inp.seq_lens, dk, dv,
                                  inp.tree_parent[:, :N].contiguous(), out, lse)
    assert st == kvshot.KVSHOT_ERR_WORKSPACE


def test_one_workspace_serves_successive_calls_and_shapes():
    """One workspace is reused by successive calls of different shapes and grids (units split into
    pieces that straddle CTAs and are merged): no call depends on what an earlier one left in it."""
    cases = [((3000, 517, 64), (4, 4, 4), True, True, 16, 32, 8, 12),   # 48 rows (spread), 3 caches
             ((700, 1300), (8, 12, 12), True, True, 64, 32, 8, 32),     # 128 rows (dense)
             ((250, 70), (1, 1, 1), False, True, 16, 32, 1, 2)]          # G = 32, contiguous
    prepared = []
    for k, (lens, levels, tree, paged, P, hq, hkv, nq) in enumerate(cases):
        spec, inp, dk, dv, q, N, Nq = _case(lens, levels, tree, paged, P, hq, hkv, nq, seed=100 + k)
        ref = gh.oracle_attn(gh.HostCache(inp), q, dk, dv, N, Nq)
        prepared.append((spec, inp, dk, dv, q, N, Nq, ref))
    ws = torch.full((64 << 20,), 0x7F, dtype=torch.uint8, device="cuda")  # not zero: nothing may be assumed
    for rep in range(2):
        for k, (spec, inp, dk, dv, q, N, Nq, (ref_out, ref_lse)) in enumerate(prepared):
            for flags in (kvshot.KVSHOT_FORCE_TC, kvshot.KVSHOT_FORCE_MMA):
                for num_ctas in (7, 3, 0):
                    out, lse = _run(spec, inp, dk, dv, q, N, Nq, flags=flags, num_ctas=num_ctas, ws=ws)
                    gh.compare(out, lse, ref_out, ref_lse, f"shared workspace rep {rep} case {k} flags {flags} ctas {num_ctas}")
