"""kvshot_draft_attn_static: draft attention for callers that cannot allocate
device memory (the scratch lives in a fixed array inside the library).

Checked through the C ABI against the CPU oracle and against the ordinary
kvshot_draft_attn on three different problems called back to back (the third
a whole tree of 64 nodes over 16 caches: 256 stacked rows per KV head on the
tcgen05 kernel's paired blocks, whose plan takes more than half of the
array), so that whatever one call left in the shared scratch array cannot
leak into the next.  This file is collected last on
purpose.
"""
import pytest
import torch

from paper_2604_26412_gb300 import kvshot
from paper_2604_26412_gb300 import workloads as wl
from tests import gpu_helpers as gh

pytestmark = pytest.mark.gpu


def _problem(lens, levels, tree, paged, page_size, n_query, seed, B=None):
    B = len(lens) if B is None else B
    spec = wl.Spec("noalloc", B, len(lens) // B, list(lens), list(levels), tree, paged, page_size=page_size,
                   seed=seed)
    inp = wl.make_inputs(spec, "cuda", seed=seed, tail_fill="nan")
    N = spec.n_nodes
    dk, dv = wl.random_draft_kv(spec, inp.n_max, N, "cuda", seed=seed + 1)
    q = wl.random_queries(spec, n_query, "cuda", seed=seed + 2)
    d = kvshot.make_desc(num_caches=spec.num_caches, num_seqs=spec.num_seqs, hq=spec.hq, hkv=spec.hkv, n_nodes=N,
                         n_query=n_query, n_max=inp.n_max, max_seq_len=spec.max_seq_len,
                         page_size=page_size if paged else 0,
                         max_pages_per_seq=inp.page_table.shape[1] if paged else 0,
                         num_pages=inp.num_pages if paged else 0, l_cap=inp.l_cap, tree=tree)
    return spec, inp, dk, dv, q, d, inp.tree_parent[:, :N].contiguous()


def _outputs(q):
    return (torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device="cuda"),
            torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device="cuda"))


def test_static_scratch_entry_point_matches_oracle_and_allocating_one():
    problems = [
        _problem((3000, 517, 64), (4, 4, 4), True, True, 16, 4, seed=31),       # tree, paged, partial pieces
        _problem((1200,), (1,) * 6, False, False, 64, 1, seed=47),               # chain, contiguous
        # whole tree of 64 nodes over 16 caches: 256 stacked rows per KV head, tcgen05 kernel, paired row blocks
        _problem((300,) * 16, (8, 12, 12, 12, 12, 8), True, True, 16, 64, seed=53, B=4),
    ]
    need = kvshot.workspace_size(problems[2][5])
    assert 32 << 20 < need <= kvshot.STATIC_WORKSPACE_BYTES, need
    static_out = []
    for spec, inp, dk, dv, q, d, par in problems:
        out, lse = _outputs(q)
        st = kvshot.draft_attn_static_status(d, q, inp.target_k, inp.target_v, inp.page_table, inp.seq_lens, dk, dv,
                                             par, out, lse)
        assert st == kvshot.KVSHOT_OK, kvshot.status_string(st)
        static_out.append((out, lse))
    torch.cuda.synchronize()
    for (spec, inp, dk, dv, q, d, par), (out_s, lse_s) in zip(problems, static_out):
        ref_out, ref_lse = gh.oracle_attn(gh.HostCache(inp), q, dk, dv, spec.n_nodes, q.shape[1])
        gh.compare(out_s, lse_s, ref_out, ref_lse, "static-scratch entry point vs the oracle")
        need = kvshot.workspace_size(d)
        assert 0 < need <= kvshot.STATIC_WORKSPACE_BYTES
        ws = torch.empty(need, dtype=torch.uint8, device="cuda")
        d.workspace, d.workspace_bytes = ws.data_ptr(), need
        out_r, lse_r = _outputs(q)
        kvshot.draft_attn(d, q, inp.target_k, inp.target_v, inp.page_table, inp.seq_lens, dk, dv, par, out_r, lse_r)
        torch.cuda.synchronize()
        gh.compare(out_s, lse_s, out_r.double().cpu().numpy(), lse_r.double().cpu().numpy(),
                   "static-scratch entry point vs kvshot_draft_attn")


def test_static_scratch_rejects_plans_larger_than_the_array():
    # 1024 caches x 8 KV heads x 256 stacked rows need more than 64 MiB of piece states.  Every data
    # pointer is NULL: were the size check ever skipped, the call would stop at KVSHOT_ERR_NULL on the host.
    d = kvshot.make_desc(num_caches=1024, num_seqs=1024, hq=32, hkv=8, n_nodes=64, n_query=64, n_max=64,
                         max_seq_len=1 << 20, page_size=16, max_pages_per_seq=1 << 16, num_pages=1 << 16, tree=True)
    assert kvshot.workspace_size(d) > kvshot.STATIC_WORKSPACE_BYTES
    st = kvshot.draft_attn_static_status(d, None, None, None, None, None, None, None, None, None, None)
    assert st == kvshot.KVSHOT_ERR_WORKSPACE
