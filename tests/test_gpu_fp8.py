"""GPU parity of kvshot_draft_attn on an fp8 (e4m3) target cache (KVSHOT_TARGET_FP8).

The target K/V are e4m3 codes with power-of-two scales; the oracle decodes them
exactly (oracle/fp8.py) to the bf16 values the kernel must use and runs the
plain attention oracle on those, so the tolerances are the bf16 path's:
out max-abs <= 2e-2, rel-L2 <= 5e-3, lse max-abs <= 1e-3.  Unused cache rows
hold NaN codes and unused draft slots NaN.
"""
import numpy as np
import pytest
import torch

from oracle import fp8 as of8
from paper_2604_26412_gb300 import kvshot
from paper_2604_26412_gb300 import workloads as wl
from tests import gpu_helpers as gh

pytestmark = pytest.mark.gpu

CASES = [
    # lens, levels, tree, paged, page_size, hq, hkv, n_query
    ((128,), (1, 1, 1, 1), False, False, 16, 32, 8, 1),          # tiny chain, contiguous
    ((0,), (1, 1, 1), False, False, 16, 32, 8, 1),                # empty prefix
    ((1, 63, 64, 65), (1, 1), False, True, 16, 32, 8, 1),         # ragged around the tile size
    ((17, 130, 300), (4, 4), True, True, 8, 32, 8, 4),            # tree, 16 rows, P = 8
    ((4096, 1000), (8, 12, 12), True, True, 16, 32, 8, 12),       # 48 rows (tcgen05 when forced: spread rows)
    ((257, 513), (8, 12, 12), True, True, 64, 32, 8, 32),         # 128 rows, row blocks
    ((700,), (2, 3, 3), True, True, 128, 32, 8, 8),               # page larger than a tile
    ((333, 5), (3, 3), True, False, 16, 8, 8, 3),                 # G = 1
    ((65,), tuple([1] * 70), False, False, 16, 4, 4, 2),          # chain with N = 70 > one draft tile
    ((203, 64), tuple([1] * 40), False, False, 16, 32, 8, 32),    # 128 dense rows, contiguous l_cap % 8 != 0
    ((300, 200), (8, 12, 12, 12), True, True, 16, 32, 8, 40),     # 160 rows: m16n8k16 only (no paired fp8 blocks)
]


def _setup(case, seed):
    lens, levels, tree, paged, P, hq, hkv, nq = case
    spec = wl.Spec("fp8", len(lens), 1, list(lens), list(levels), tree, paged, page_size=P, hq=hq, hkv=hkv, seed=seed)
    inp = wl.make_inputs(spec, "cuda", seed=seed, tail_fill="nan")
    N = spec.n_nodes
    dk, dv = wl.random_draft_kv(spec, inp.n_max, N, "cuda", seed=seed + 1, tail=float("nan"))
    q = wl.random_queries(spec, nq, "cuda", seed=seed + 2)
    tk8, tv8 = wl.fp8_target(inp)
    hc = gh.HostCache(inp)
    hc.tk = of8.dequant_bf16_bits(tk8.cpu().numpy(), wl.FP8_K_EXP)
    hc.tv = of8.dequant_bf16_bits(tv8.cpu().numpy(), wl.FP8_V_EXP)
    return spec, inp, dk, dv, q, N, nq, tk8, tv8, hc


def _run(spec, inp, tk8, tv8, dk, dv, q, N, Nq, flags, num_ctas=0):
    paged = inp.page_table is not None
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = kvshot.make_desc(num_caches=spec.num_caches, num_seqs=spec.num_seqs, hq=spec.hq, hkv=spec.hkv, n_nodes=N,
                         n_query=Nq, n_max=inp.n_max, max_seq_len=spec.max_seq_len,
                         page_size=spec.page_size if paged else 0,
                         max_pages_per_seq=inp.page_table.shape[1] if paged else 0,
                         num_pages=inp.num_pages if paged else 0, l_cap=inp.l_cap, tree=spec.tree,
                         flags=flags | kvshot.KVSHOT_TARGET_FP8, num_ctas=num_ctas, err_flag=err,
                         k_scale_exp=wl.FP8_K_EXP, v_scale_exp=wl.FP8_V_EXP)
    ws = torch.empty(kvshot.workspace_size(d), dtype=torch.uint8, device="cuda")
    d.workspace, d.workspace_bytes = ws.data_ptr(), ws.numel()
    kvshot.draft_attn(d, q, tk8, tv8, inp.page_table, inp.seq_lens, dk, dv, inp.tree_parent[:, :N].contiguous(),
                      out, lse)
    torch.cuda.synchronize()
    assert int(err.item()) == 0, f"device error {int(err.item())}"
    return out, lse


@pytest.mark.parametrize("case", CASES, ids=[f"c{i}" for i in range(len(CASES))])
def test_fp8_target_matches_oracle(case):
    spec, inp, dk, dv, q, N, Nq, tk8, tv8, hc = _setup(case, seed=3 + len(case[0]) + sum(case[1]))
    ref_out, ref_lse = gh.oracle_attn(hc, q, dk, dv, N, Nq)
    rows = case[5] // case[6] * case[7]
    for flags in (0, kvshot.KVSHOT_FORCE_MMA) + ((kvshot.KVSHOT_FORCE_TC,) if rows <= 128 else ()):
        for num_ctas in (0, 1, 7):
            out, lse = _run(spec, inp, tk8, tv8, dk, dv, q, N, Nq, flags, num_ctas)
            gh.compare(out, lse, ref_out, ref_lse, f"fp8 {case} flags={flags} ctas={num_ctas}")


@pytest.mark.parametrize("nq", [12, 32])
def test_fp8_tcgen05_matches_oracle_at_48_and_128_rows(nq):
    # The tcgen05 kernel decoding fp8 tiles: 48 stacked rows (spread) and 128 (dense), paged P = 16.
    case = ((3000, 517, 64), (8, 12, 12), True, True, 16, 32, 8, nq)
    spec, inp, dk, dv, q, N, Nq, tk8, tv8, hc = _setup(case, seed=nq)
    ref_out, ref_lse = gh.oracle_attn(hc, q, dk, dv, N, Nq)
    for num_ctas in (0, 3, 152):
        out, lse = _run(spec, inp, tk8, tv8, dk, dv, q, N, Nq, kvshot.KVSHOT_FORCE_TC, num_ctas)
        gh.compare(out, lse, ref_out, ref_lse, f"fp8 tcgen05 nq={nq} ctas={num_ctas}")


def test_fp8_is_deterministic_and_differs_from_bf16_only_by_quantisation():
    spec, inp, dk, dv, q, N, Nq, tk8, tv8, hc = _setup(((2000, 900), (4, 4), True, True, 16, 32, 8, 4), seed=21)
    a = _run(spec, inp, tk8, tv8, dk, dv, q, N, Nq, 0)
    b = _run(spec, inp, tk8, tv8, dk, dv, q, N, Nq, 0)
    assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])
    # the same call on the bf16 cache the codes were made from: close, but not equal (quantisation)
    hb = gh.HostCache(inp)
    ref_bf16, _ = gh.oracle_attn(hb, q, dk, dv, N, Nq)
    o = a[0].float().cpu().numpy().astype(np.float64)
    rel = np.linalg.norm(o - ref_bf16) / np.linalg.norm(ref_bf16)
    assert 1e-3 < rel < 0.1, rel
