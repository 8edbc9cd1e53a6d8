"""GPU parity of the draft append with QK-norm (kvshot_draft_append_qknorm) with the fp64 oracle.

The kernel normalises and rotates in fp32 and rounds once to bf16, so every
q and k element is within one bf16 rounding step of the fp64 value plus the
fp32 error of a unit-RMS head: |gpu - oracle| <= 2^-8 |oracle| + 1e-5 (the
fp32 error of a 128-term mean square, rsqrt and rotation is a few 2^-24
times the head's largest value, which the weights keep below ~4), and nearly
every element (>= 99%) carries exactly the bits of the fp64 value rounded to
nearest.  Values are copied, so V must match bit for bit; slots outside
n0 .. n0 + n_new - 1 must be left as they were.
"""
import numpy as np
import pytest
import torch

from oracle import qknorm as qo
from paper_2604_26412_gb300 import kvshot
from paper_2604_26412_gb300 import workloads as wl
from tests.gpu_helpers import round_bf16_bits as _round_bf16, widen_bits as _widen

pytestmark = pytest.mark.gpu
D = 128


def _case(C, hq, hkv, n_new, n0, n_max, max_pos, seed, in_place=False, eps=1e-6):
    g = torch.Generator().manual_seed(seed)
    q_in = (torch.randn((C, n_new, hq, D), generator=g) * 3).to(torch.bfloat16)
    k_in = (torch.randn((C, n_new, hkv, D), generator=g) * 3).to(torch.bfloat16)
    v_in = torch.randn((C, n_new, hkv, D), generator=g).to(torch.bfloat16)
    pos = torch.randint(0, max_pos, (C, n_new), generator=g, dtype=torch.int32)
    wq = (0.5 + 1.5 * torch.rand(D, generator=g)).to(torch.bfloat16)
    wk = (0.5 + 1.5 * torch.rand(D, generator=g)).to(torch.bfloat16)
    dk0 = torch.randn((C, hkv, n_max, D), generator=g).to(torch.bfloat16)
    dv0 = torch.randn((C, hkv, n_max, D), generator=g).to(torch.bfloat16)
    dev = [t.cuda() for t in (q_in, k_in, v_in, pos, wq, wk, dk0, dv0)]
    q_d, k_d, v_d, p_d, wq_d, wk_d, dk, dv = dev
    q_out = q_d if in_place else torch.empty_like(q_d)
    base = 1e6
    d = kvshot.make_desc(num_caches=C, num_seqs=C, hq=hq, hkv=hkv, n_nodes=0, n_query=0, n_max=n_max, max_seq_len=0)
    kvshot.draft_append_qknorm(d, q_d, k_d, v_d, p_d, n0, n_new, base, wq_d, wk_d, eps, dk, dv, q_out)
    torch.cuda.synchronize()
    qr, kr, vr = qo.append_qknorm(wl.bf16_bits(q_in), wl.bf16_bits(k_in), wl.bf16_bits(v_in), pos.numpy(), n0, base,
                                  wl.bf16_bits(wq), wl.bf16_bits(wk), eps, n_max)
    gq, gk, gv = wl.bf16_bits(q_out), wl.bf16_bits(dk), wl.bf16_bits(dv)
    exact = 0
    total = 0
    for got, ref, what in ((gq, qr, "q"), (gk[:, :, n0:n0 + n_new], kr, "k")):
        gf = _widen(got)
        assert np.all(np.isfinite(gf)), what
        err = np.abs(gf - ref)
        bound = 2.0 ** -8 * np.abs(ref) + 1e-5
        assert np.all(err <= bound), f"{what}: worst excess {np.max(err - bound):.3g}"
        exact += int(np.sum(got == _round_bf16(ref)))
        total += got.size
    assert exact >= 0.99 * total, f"only {exact} of {total} elements rounded like the fp64 value"
    assert np.array_equal(gv[:, :, n0:n0 + n_new], wl.bf16_bits(v_in).transpose(0, 2, 1, 3))
    outside = np.ones(n_max, dtype=bool)
    outside[n0:n0 + n_new] = False
    assert np.array_equal(gk[:, :, outside], wl.bf16_bits(dk0)[:, :, outside])
    assert np.array_equal(gv[:, :, outside], wl.bf16_bits(dv0)[:, :, outside])


@pytest.mark.parametrize("C,hq,hkv,n_new,n0,n_max,max_pos", [
    (4, 32, 8, 5, 3, 16, 40000),      # one drafting level at long positions
    (2, 32, 8, 64, 0, 64, 8192),      # whole tree in one call, draft region full
    (3, 8, 1, 1, 15, 16, 100),        # one node into the last slot, MQA
    (1, 64, 4, 7, 2, 12, 1 << 20),    # more query heads than warps cover in one pass
])
def test_qknorm_append_matches_oracle(C, hq, hkv, n_new, n0, n_max, max_pos):
    _case(C, hq, hkv, n_new, n0, n_max, max_pos, seed=C * 1000 + n_new)


def test_qknorm_append_in_place():
    _case(2, 32, 8, 6, 1, 8, 30000, seed=11, in_place=True)


def test_qknorm_append_large_eps():
    # eps comparable to the mean square: the norm no longer reaches unit RMS; same bounds hold
    _case(2, 16, 4, 3, 0, 4, 500, seed=12, eps=4.0)


def test_qknorm_append_zero_nodes_is_a_no_op():
    d = kvshot.make_desc(num_caches=1, num_seqs=1, hq=8, hkv=1, n_nodes=0, n_query=0, n_max=4, max_seq_len=0)
    w = torch.ones(D, dtype=torch.bfloat16, device="cuda")
    dk = torch.full((1, 1, 4, D), 2.0, dtype=torch.bfloat16, device="cuda")
    x = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    kvshot.draft_append_qknorm(d, x, x, x, x, 0, 0, 1e6, w, w, 1e-6, dk, dk, x)
    torch.cuda.synchronize()
    assert bool((dk == 2.0).all())
