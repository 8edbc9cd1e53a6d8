"""GPU parity of the gated-delta fusion (kvshot_gated_delta) with the fp64 oracle.

Tolerance.  The library accumulates in fp32 (K = d to 3d terms of O(1)
products: relative error ~1e-6) and rounds h once to bf16 (at most 2^-9 of
|h|).  Every element must satisfy |gpu - oracle| <= 2^-8 |oracle| + 1e-3 (one
bf16 ulp plus the fp32 accumulation), and the relative L2 error over the
output must be <= 3e-3.
"""
import numpy as np
import pytest
import torch

from oracle import fusion as fo
from paper_2604_26412_gb300 import kvshot
from paper_2604_26412_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def _run(fi, T, d, ws=None, err=None):
    desc = kvshot.make_fusion_desc(num_tokens=T, hidden=d)
    need = kvshot.gated_delta_workspace_size(desc)
    assert need > 0
    if ws is None:
        ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    desc.workspace, desc.workspace_bytes = ws.data_ptr(), ws.numel()
    err = torch.zeros(1, dtype=torch.int32, device="cuda") if err is None else err
    desc.err_flag = err.data_ptr()
    h = torch.full((T, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    kvshot.gated_delta(desc, fi.n, fi.o, fi.w_g, fi.b_g, fi.w_delta, h)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    return h


def _oracle(fi):
    bits = lambda t: wl.bf16_bits(t.cpu())
    return fo.gated_delta(bits(fi.n), bits(fi.o), bits(fi.w_g), bits(fi.b_g), bits(fi.w_delta))


def _compare(h, ref, what):
    got = h.double().cpu().numpy()
    assert np.isfinite(got).all(), what
    err = np.abs(got - ref)
    bound = 2.0 ** -8 * np.abs(ref) + 1e-3
    worst = np.argmax(err - bound)
    assert (err <= bound).all(), f"{what}: element {np.unravel_index(worst, ref.shape)} |err| {err.flat[worst]:.3g}"
    rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
    assert rel <= 3e-3, f"{what}: relative L2 error {rel:.3g}"


# (T, d): one token; token counts that are and are not multiples of 16; 128 and 129 tokens (the
# largest block whose n and o rows stack into one MMA, and one past it: negated-weight MMAs); 256
# (a full block) and 257 (a second block of one token); d from 128 to 1024.
@pytest.mark.parametrize("T,d", [(1, 128), (5, 256), (16, 384), (127, 512), (128, 256), (129, 384), (192, 1024),
                                 (300, 512), (256, 640), (257, 128)])
def test_fusion_matches_oracle(T, d):
    fi = wl.fusion_inputs(T, d, device="cuda", seed=T + d)
    _compare(_run(fi, T, d), _oracle(fi), f"T={T} d={d}")


def test_fusion_full_width_hybrid_tree_level():
    # The hybrid-tree workload's widest per-depth step: 16 sequences x 12 draft nodes, d = 4096.
    T, d = 16 * 12, wl.HIDDEN
    fi = wl.fusion_inputs(T, d, device="cuda", seed=11)
    _compare(_run(fi, T, d), _oracle(fi), "hybrid tree level, d=4096")


def test_no_correction_when_branches_agree_is_exact():
    # o = n: W o and W n are the same tensor-core sums, so delta's products cancel exactly and h == n bit for bit.
    T, d = 40, 512
    fi = wl.fusion_inputs(T, d, device="cuda", seed=3)
    fi.o = fi.n.clone()
    h = _run(fi, T, d)
    assert torch.equal(h, fi.n)


def test_gate_extremes():
    T, d = 24, 256
    fi = wl.fusion_inputs(T, d, device="cuda", seed=4)
    fi.w_g = torch.zeros_like(fi.w_g)
    fi.w_delta = torch.eye(d, dtype=torch.bfloat16, device="cuda")
    fi.b_g = torch.full((d,), 40.0, dtype=torch.bfloat16, device="cuda")   # g = 1: h = n + (o - n) = o
    _compare(_run(fi, T, d), _oracle(fi), "open gate")
    assert torch.allclose(_run(fi, T, d).float(), fi.o.float(), atol=2e-2, rtol=2 ** -8)
    fi.b_g = torch.full((d,), -40.0, dtype=torch.bfloat16, device="cuda")  # g = 0: h = n
    assert torch.equal(_run(fi, T, d), fi.n)


def test_workspace_reuse_and_garbage():
    # The workspace needs no initialisation: fill it with NaN bit patterns and reuse it across shapes.
    shapes = ((300, 512), (7, 1024), (130, 256))
    need = max(kvshot.gated_delta_workspace_size(kvshot.make_fusion_desc(num_tokens=T, hidden=d)) for T, d in shapes)
    ws = torch.full((need,), 0xFF, dtype=torch.uint8, device="cuda")
    for T, d in shapes:
        fi = wl.fusion_inputs(T, d, device="cuda", seed=T)
        _compare(_run(fi, T, d, ws=ws), _oracle(fi), f"reused workspace T={T} d={d}")
