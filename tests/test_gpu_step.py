"""GPU parity of the whole hot path (append + attention, every drafting level)
on the benchmark workloads at full size, against the oracle's own append and
attention.  The largest workload is checked on sampled caches."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2604_26412_gb300 import kvshot
from paper_2604_26412_gb300 import workloads as wl
from paper_2604_26412_gb300.step import DraftStep
from tests import gpu_helpers as gh

pytestmark = pytest.mark.gpu


def _oracle_step(inp, hc, mode, caches):
    """Oracle append + attention for every level, on the given caches."""
    s = inp.spec
    C = s.num_caches
    dk = np.full((C, s.hkv, inp.n_max, s.head_dim), 0x7FC0, np.uint16)
    dv = dk.copy()
    if mode == "per_depth":
        levels = list(s.levels)
        qs, ks, vs, ps = inp.q_in, inp.k_in, inp.v_in, inp.positions
    else:
        levels = [s.n_nodes]
        qs = [torch.cat(inp.q_in, 1)]
        ks = [torch.cat(inp.k_in, 1)]
        vs = [torch.cat(inp.v_in, 1)]
        ps = [torch.cat(inp.positions, 1)]
    d_app = oracle.make_desc(num_caches=C, num_seqs=s.num_seqs, hq=s.hq, hkv=s.hkv, head_dim=s.head_dim, n_nodes=0,
                             n_query=0, n_max=inp.n_max, tree=s.tree, l_cap=1)
    results = []
    n0 = 0
    for i, n_step in enumerate(levels):
        q_rot = oracle.append(d_app, wl.bf16_bits(qs[i]), wl.bf16_bits(ks[i]), wl.bf16_bits(vs[i]),
                              ps[i].cpu().numpy(), n0, n_step, s.rope_base, dk, dv)
        n0 += n_step
        out, lse = gh.oracle_attn(hc, wl.bits_to_bf16(q_rot), wl.bits_to_bf16(dk), wl.bits_to_bf16(dv), n0, n_step,
                                  caches=caches)
        results.append((out, lse, q_rot, dk.copy()))
    return results


@pytest.mark.parametrize("cfg,mode,caches", [
    (1, "per_depth", None),
    (2, "per_depth", None),
    (2, "whole", None),
    (3, "per_depth", None),
    (3, "whole", [0, 5, 15]),
    (4, "per_depth", None),
    (5, "per_depth", [0, 6, 15]),
    (5, "whole", [3, 12]),
])
def test_step_matches_oracle(cfg, mode, caches):
    spec = wl.config(cfg, seed=0)
    inp = wl.make_inputs(spec, "cuda")
    step = DraftStep(inp, mode=mode)
    step.run()
    torch.cuda.synchronize()
    assert step.error_code() == 0
    hc = gh.HostCache(inp)
    ref = _oracle_step(inp, hc, mode, caches)
    sel = list(range(spec.num_caches)) if caches is None else caches
    for i, (ro, rl, q_rot, dk_ref) in enumerate(ref):
        # The append is exact: identical bf16 bits to the oracle's fp64 RoPE rounded once.
        assert np.array_equal(wl.bf16_bits(step.q_rot[i]), q_rot), f"level {i}: q RoPE bits differ"
        gh.compare(step.out[i][sel], step.lse[i][sel], ro, rl, f"cfg{cfg} {mode} level {i}")
    n = spec.n_nodes
    assert np.array_equal(wl.bf16_bits(step.draft_k)[:, :, :n], ref[-1][3][:, :, :n])


def test_append_is_bit_exact_at_long_positions():
    spec = wl.config(5, seed=1)
    C, D = spec.num_caches, spec.head_dim
    g = torch.Generator(device="cuda").manual_seed(7)
    n_new, n_max, n0 = 5, 16, 3
    q_in = torch.randn((C, n_new, spec.hq, D), generator=g, device="cuda").to(torch.bfloat16)
    k_in = torch.randn((C, n_new, spec.hkv, D), generator=g, device="cuda").to(torch.bfloat16)
    v_in = torch.randn((C, n_new, spec.hkv, D), generator=g, device="cuda").to(torch.bfloat16)
    pos = torch.randint(0, 40000, (C, n_new), generator=g, device="cuda", dtype=torch.int32)
    dk = torch.full((C, spec.hkv, n_max, D), 3.0, dtype=torch.bfloat16, device="cuda")
    dv = dk.clone()
    q_out = torch.empty_like(q_in)
    d = kvshot.make_desc(num_caches=C, num_seqs=spec.num_seqs, hq=spec.hq, hkv=spec.hkv, n_nodes=0, n_query=0,
                         n_max=n_max, max_seq_len=0)
    kvshot.draft_append(d, q_in, k_in, v_in, pos, n0, n_new, spec.rope_base, dk, dv, q_out)
    torch.cuda.synchronize()
    od = oracle.make_desc(num_caches=C, num_seqs=spec.num_seqs, hq=spec.hq, hkv=spec.hkv, head_dim=D, n_nodes=0,
                          n_query=0, n_max=n_max, tree=False, l_cap=1)
    dk_ref = np.full((C, spec.hkv, n_max, D), wl.bf16_bits(torch.tensor([3.0], dtype=torch.bfloat16))[0], np.uint16)
    dv_ref = dk_ref.copy()
    q_ref = oracle.append(od, wl.bf16_bits(q_in), wl.bf16_bits(k_in), wl.bf16_bits(v_in), pos.cpu().numpy(), n0,
                          n_new, spec.rope_base, dk_ref, dv_ref)
    assert np.array_equal(wl.bf16_bits(q_out), q_ref)
    assert np.array_equal(wl.bf16_bits(dk), dk_ref)
    assert np.array_equal(wl.bf16_bits(dv), dv_ref)
    # in place (q_out == q_in) gives the same bits
    kvshot.draft_append(d, q_in, k_in, v_in, pos, n0, n_new, spec.rope_base, dk, dv, q_in)
    torch.cuda.synchronize()
    assert np.array_equal(wl.bf16_bits(q_in), q_ref)


@pytest.mark.parametrize("cfg,caches", [(2, None), (5, [1, 10])])
def test_step_with_qknorm_matches_oracle(cfg, caches):
    """The step with the QK-norm append (kvshot_draft_append_qknorm) against the oracle's QK-norm append and
    attention.  The append rounds once from fp32, so q and k are within one bf16 step of the fp64 values; the
    attention is held to the usual tolerances on the oracle's own rounded q and k."""
    from oracle import qknorm as qo
    spec = wl.config(cfg, seed=0)
    inp = wl.make_inputs(spec, "cuda")
    g = torch.Generator().manual_seed(23)
    wq = (0.5 + torch.rand(spec.head_dim, generator=g)).to(torch.bfloat16)
    wk = (0.5 + torch.rand(spec.head_dim, generator=g)).to(torch.bfloat16)
    eps = 1e-6
    step = DraftStep(inp, mode="per_depth", qk_norm=(wq.cuda(), wk.cuda(), eps))
    step.run()
    torch.cuda.synchronize()
    assert step.error_code() == 0
    hc = gh.HostCache(inp)
    sel = list(range(spec.num_caches)) if caches is None else caches
    C, D = spec.num_caches, spec.head_dim
    dk = np.full((C, spec.hkv, inp.n_max, D), 0x7FC0, np.uint16)
    dv = dk.copy()
    n0 = 0
    for i, n_step in enumerate(spec.levels):
        qr, kr, vr = qo.append_qknorm(wl.bf16_bits(inp.q_in[i]), wl.bf16_bits(inp.k_in[i]), wl.bf16_bits(inp.v_in[i]),
                                      inp.positions[i].cpu().numpy(), n0, spec.rope_base, wl.bf16_bits(wq),
                                      wl.bf16_bits(wk), eps, inp.n_max)
        dk[:, :, n0:n0 + n_step] = gh.round_bf16_bits(kr)
        dv[:, :, n0:n0 + n_step] = gh.round_bf16_bits(vr)
        n0 += n_step
        gq = gh.widen_bits(wl.bf16_bits(step.q_rot[i]))
        assert np.all(np.abs(gq - qr) <= 2.0 ** -8 * np.abs(qr) + 1e-5), f"level {i}: q off by more than a bf16 step"
        out, lse = gh.oracle_attn(hc, wl.bits_to_bf16(gh.round_bf16_bits(qr)), wl.bits_to_bf16(dk),
                                  wl.bits_to_bf16(dv), n0, n_step, caches=caches)
        gh.compare(step.out[i][sel], step.lse[i][sel], out, lse, f"cfg{cfg} qk-norm level {i}")
    gk = gh.widen_bits(wl.bf16_bits(step.draft_k)[:, :, :n0])
    rk = gh.widen_bits(dk[:, :, :n0])
    assert np.all(np.abs(gk - rk) <= 2.0 ** -7 * np.abs(rk) + 1e-5)
    assert np.array_equal(wl.bf16_bits(step.draft_v)[:, :, :n0], dv[:, :, :n0])
