"""GPU parity of the multi-layer KV projection (kvshot_kv_project) with the fp64 oracle.

Tolerance as for the fusion: fp32 accumulation over L d_kv terms and one bf16
rounding, so |gpu - oracle| <= 2^-8 |oracle| + 1e-3 per element and relative
L2 <= 3e-3 over the written rows.  Rows the call does not own must be left
bit for bit as they were.
"""
import numpy as np
import pytest
import torch

from oracle import project as po
from paper_2604_26412_gb300 import kvshot
from paper_2604_26412_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
D = 128


def _pool_layout(C, hkv, paged, P, cap_tokens, rng):
    if paged:
        pages_per = (cap_tokens + P - 1) // P
        num_pages = C * pages_per + 3
        pt = rng.permutation(num_pages)[:C * pages_per].reshape(C, pages_per).astype(np.int32)
        rows = num_pages * hkv * P
        return dict(page_table=pt, num_pages=num_pages, page_size=P, max_pages=pages_per, rows=rows, l_cap=0)
    return dict(page_table=None, num_pages=0, page_size=0, max_pages=0, rows=C * hkv * cap_tokens, l_cap=cap_tokens)


def _run_case(T, L, hkv, C, paged, P, cap, rope, seed):
    rng = np.random.default_rng(seed)
    pi = wl.project_inputs(T, L, hkv, device="cuda", seed=seed)
    lay = _pool_layout(C, hkv, paged, P, cap, rng)
    # distinct (cache, position) slots
    flat = rng.choice(C * cap, size=T, replace=False)
    token_cache, positions = (flat // cap).astype(np.int32), (flat % cap).astype(np.int32)
    k_pool = torch.randn((lay["rows"], D), device="cuda").to(torch.bfloat16)
    v_pool = torch.randn((lay["rows"], D), device="cuda").to(torch.bfloat16)
    k0, v0 = k_pool.clone(), v_pool.clone()
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = kvshot.make_project_desc(num_tokens=T, num_layers=L, hkv=hkv, num_caches=C, page_size=lay["page_size"],
                                 max_pages_per_seq=lay["max_pages"], num_pages=lay["num_pages"], l_cap=lay["l_cap"],
                                 rope=rope, err_flag=err)
    ws = torch.empty(max(256, kvshot.kv_project_workspace_size(d)), dtype=torch.uint8, device="cuda")
    d.workspace, d.workspace_bytes = ws.data_ptr(), ws.numel()
    tc, ps = torch.from_numpy(token_cache).cuda(), torch.from_numpy(positions).cuda()
    pt = torch.from_numpy(lay["page_table"]).cuda() if paged else None
    kvshot.kv_project(d, pi.k_in, pi.v_in, pi.w_k, pi.w_v, tc, ps, pt, k_pool, v_pool)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    bits = lambda t: wl.bf16_bits(t.cpu())
    kref, vref = po.kv_project(bits(pi.k_in), bits(pi.v_in), bits(pi.w_k), bits(pi.w_v), positions, 1.0e6, rope)
    rows = po.cache_rows(token_cache, positions, hkv, page_table=lay["page_table"], page_size=P, l_cap=lay["l_cap"])
    return k_pool, v_pool, k0, v0, kref.reshape(T, hkv, D), vref.reshape(T, hkv, D), rows


def _check(pool, pool0, ref, rows, what):
    got = pool.double().cpu().numpy()[rows]  # [T, hkv, D]
    err = np.abs(got - ref)
    assert (err <= 2.0 ** -8 * np.abs(ref) + 1e-3).all(), f"{what}: max err {err.max():.3g}"
    assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 3e-3, what
    mask = torch.ones(pool.shape[0], dtype=torch.bool)
    mask[torch.from_numpy(rows.reshape(-1))] = False
    assert torch.equal(pool.cpu()[mask], pool0.cpu()[mask]), f"{what}: rows outside the call changed"


@pytest.mark.parametrize("T,L,hkv,C,paged,P,cap,rope", [
    (1, 1, 1, 1, False, 0, 8, True),
    (7, 3, 2, 3, True, 16, 64, True),
    (64, 3, 8, 16, True, 16, 256, True),
    (64, 3, 8, 16, True, 16, 256, False),
    (130, 2, 4, 5, False, 0, 300, True),
    (33, 4, 8, 4, True, 64, 512, True),
    (9, 5, 2, 2, False, 0, 40, True),       # 5 layers: K ranges not split (table of 16 entries)
])
def test_projection_matches_oracle(T, L, hkv, C, paged, P, cap, rope):
    k_pool, v_pool, k0, v0, kref, vref, rows = _run_case(T, L, hkv, C, paged, P, cap, rope, seed=T + L + hkv)
    _check(k_pool, k0, kref, rows, "K")
    _check(v_pool, v0, vref, rows, "V")


def test_out_of_range_slot_is_reported_and_skipped():
    T, L, hkv, C, cap = 4, 2, 2, 2, 16
    pi = wl.project_inputs(T, L, hkv, device="cuda", seed=3)
    k_pool = torch.zeros((C * hkv * cap, D), dtype=torch.bfloat16, device="cuda")
    v_pool = torch.zeros_like(k_pool)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = kvshot.make_project_desc(num_tokens=T, num_layers=L, hkv=hkv, num_caches=C, l_cap=cap, err_flag=err)
    ws = torch.empty(kvshot.kv_project_workspace_size(d), dtype=torch.uint8, device="cuda")
    d.workspace, d.workspace_bytes = ws.data_ptr(), ws.numel()
    tc = torch.tensor([0, 1, 5, 0], dtype=torch.int32, device="cuda")      # cache 5 does not exist
    ps = torch.tensor([0, 3, 1, 99], dtype=torch.int32, device="cuda")     # position 99 >= l_cap
    kvshot.kv_project(d, pi.k_in, pi.v_in, pi.w_k, pi.w_v, tc, ps, None, k_pool, v_pool)
    torch.cuda.synchronize()
    assert int(err.item()) == kvshot.KVSHOT_ERR_DEVICE_BOUNDS
    written = (k_pool.float().abs().sum(dim=1) > 0).nonzero().flatten().tolist()
    expect = sorted(((0 * hkv + h) * cap + 0) for h in range(hkv)) + sorted(((1 * hkv + h) * cap + 3) for h in range(hkv))
    assert sorted(written) == sorted(expect)
