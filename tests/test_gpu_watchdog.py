"""The attention kernels' pipeline watchdog, exercised on the GPU without a fault.

desc.wait_limit_ns bounds every wait of the load/compute pipeline.  With a
limit of 1 ns each CTA gives up on the first wait whose data has not arrived
yet: the call must still end (the abort drains the copies and tensor-core
operations already issued, with the ordinary 2 s limit), record
KVSHOT_ERR_TIMEOUT in err_flag, and leave the stream, the device and the
workspace fit for the next call, which must match the CPU oracle.  Every
kernel is driven through its abort path: tcgen05 with spread, dense and paired rows,
m16n8k16 and the CUDA-core kernel.
"""
import pytest
import torch

from paper_2604_26412_gb300 import kvshot
from paper_2604_26412_gb300 import workloads as wl
from tests import gpu_helpers as gh

pytestmark = pytest.mark.gpu


def _problem(n_query, seed):
    spec = wl.Spec("watchdog", 3, 1, [3000, 517, 64], [8, 12, 12, 12], True, True, page_size=16, seed=seed)
    inp = wl.make_inputs(spec, "cuda", seed=seed, tail_fill="nan")
    N = spec.n_nodes
    dk, dv = wl.random_draft_kv(spec, inp.n_max, N, "cuda", seed=seed + 1)
    q = wl.random_queries(spec, n_query, "cuda", seed=seed + 2)
    return spec, inp, dk, dv, q, N


def _call(spec, inp, dk, dv, q, N, flags, wait_limit_ns, ws):
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = kvshot.make_desc(num_caches=spec.num_caches, num_seqs=spec.num_seqs, hq=spec.hq, hkv=spec.hkv, n_nodes=N,
                         n_query=q.shape[1], n_max=inp.n_max, max_seq_len=spec.max_seq_len,
                         page_size=spec.page_size, max_pages_per_seq=inp.page_table.shape[1],
                         num_pages=inp.num_pages, tree=True, flags=flags, err_flag=err,
                         wait_limit_ns=wait_limit_ns)
    need = kvshot.workspace_size(d)
    assert 0 < need <= ws.numel()
    d.workspace, d.workspace_bytes = ws.data_ptr(), ws.numel()
    out = torch.full(q.shape, float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device="cuda")
    st = kvshot.draft_attn_status(d, q, inp.target_k, inp.target_v, inp.page_table, inp.seq_lens, dk, dv,
                                  inp.tree_parent[:, :N].contiguous(), out, lse)
    assert st == kvshot.KVSHOT_OK, kvshot.status_string(st)
    torch.cuda.synchronize()
    return int(err.item()), out, lse


@pytest.mark.parametrize("flags,n_query", [
    (kvshot.KVSHOT_FORCE_TC, 12),    # 48 rows: spread TMEM rows
    (kvshot.KVSHOT_FORCE_TC, 32),    # 128 rows: dense TMEM rows
    (kvshot.KVSHOT_FORCE_TC, 40),    # 160 rows: paired row blocks
    (kvshot.KVSHOT_FORCE_MMA, 4),
    (kvshot.KVSHOT_FORCE_CC, 4),
])
def test_watchdog_timeout_is_reported_and_the_next_call_is_correct(flags, n_query):
    spec, inp, dk, dv, q, N = _problem(n_query, seed=41 + n_query)
    ws = torch.empty(64 << 20, dtype=torch.uint8, device="cuda")
    for _ in range(2):  # twice in a row: an aborted call leaves nothing behind that blocks the next one
        code, _, _ = _call(spec, inp, dk, dv, q, N, flags, 1, ws)
        assert code == kvshot.KVSHOT_ERR_TIMEOUT, code
    code, out, lse = _call(spec, inp, dk, dv, q, N, flags, 0, ws)
    assert code == 0, code
    ref_out, ref_lse = gh.oracle_attn(gh.HostCache(inp), q, dk, dv, N, q.shape[1])
    gh.compare(out, lse, ref_out, ref_lse, f"after a timed-out call, flags={flags}")
