"""Pins for the oracle's draft append (RoPE + slot store) and its bf16 rounding (no GPU)."""
import math

import numpy as np
import pytest
import torch

from paper_2604_26412_gb300 import workloads as wl
from tests import brute, problems


def _append_case(oracle_mod, positions, D=128, hq=4, hkv=2, base=1e6, n0=3, seed=0):
    C, n_new = positions.shape
    spec = problems.small_spec(B=C, lens=(4,) * C, levels=(n0 + n_new,), hq=hq, hkv=hkv, D=D)
    g = torch.Generator().manual_seed(seed)
    q_in = torch.randn((C, n_new, hq, D), generator=g).to(torch.bfloat16)
    k_in = torch.randn((C, n_new, hkv, D), generator=g).to(torch.bfloat16)
    v_in = torch.randn((C, n_new, hkv, D), generator=g).to(torch.bfloat16)
    n_max = n0 + n_new + 2
    dk, dv = wl.draft_buffers(spec, n_max, "cpu", fill=7.0)
    dk, dv = wl.bf16_bits(dk).copy(), wl.bf16_bits(dv).copy()
    d = oracle_mod.make_desc(num_caches=C, num_seqs=C, hq=hq, hkv=hkv, head_dim=D, n_nodes=0, n_query=0,
                             n_max=n_max, tree=False, l_cap=4)
    qb, kb, vb = wl.bf16_bits(q_in), wl.bf16_bits(k_in), wl.bf16_bits(v_in)
    q_out, q_rot, k_rot = oracle_mod.append(d, qb, kb, vb, positions, n0, n_new, base, dk, dv, want_f64=True)
    return dict(qb=qb, kb=kb, vb=vb, q_out=q_out, q_rot=q_rot, k_rot=k_rot, dk=dk, dv=dv, n0=n0, n_new=n_new,
                D=D, base=base, positions=positions)


def _complex_rope(x, pos, base):
    """Textbook RoPE as complex multiplication: z_j = x_j + i x_{j+D/2} times exp(i pos w_j)."""
    D = x.shape[-1]
    half = D // 2
    w = base ** (-np.arange(half) * 2.0 / D)
    z = (x[..., :half] + 1j * x[..., half:]) * np.exp(1j * pos * w)
    return np.concatenate([z.real, z.imag], axis=-1)


def test_rope_matches_complex_rotation(oracle_mod):
    pos = np.array([[0, 1, 4099], [32775, 17, 2]], np.int32)
    r = _append_case(oracle_mod, pos)
    qf, kf = brute.bits_to_f64(r["qb"]), brute.bits_to_f64(r["kb"])
    for c in range(2):
        for i in range(3):
            np.testing.assert_allclose(r["q_rot"][c, i], _complex_rope(qf[c, i], pos[c, i], 1e6), atol=1e-11)
            np.testing.assert_allclose(r["k_rot"][c, i], _complex_rope(kf[c, i], pos[c, i], 1e6), atol=1e-11)


def test_rope_position_zero_is_identity_and_norms_are_kept(oracle_mod):
    pos = np.array([[0, 5, 1000]], np.int32)
    r = _append_case(oracle_mod, pos, D=16, base=10000.0)
    qf = brute.bits_to_f64(r["qb"])
    assert np.array_equal(r["q_rot"][0, 0], qf[0, 0])
    half = 8
    for i in range(3):
        a, b = qf[0, i, :, :half], qf[0, i, :, half:]
        ra, rb = r["q_rot"][0, i, :, :half], r["q_rot"][0, i, :, half:]
        np.testing.assert_allclose(ra ** 2 + rb ** 2, a ** 2 + b ** 2, rtol=1e-13)


def test_rope_scores_depend_only_on_relative_position(oracle_mod):
    """<RoPE(q, m), RoPE(k, n)> is a function of m - n (the reason RoPE is re-applied)."""
    D = 32
    pos1 = np.array([[100, 90]], np.int32)
    pos2 = np.array([[2100, 2090]], np.int32)
    r1 = _append_case(oracle_mod, pos1, D=D, hq=2, hkv=2, seed=4)
    r2 = _append_case(oracle_mod, pos2, D=D, hq=2, hkv=2, seed=4)
    # q at node 0 (pos m), k at node 1 (pos n)
    s1 = r1["q_rot"][0, 0, 0] @ r1["k_rot"][0, 1, 0]
    s2 = r2["q_rot"][0, 0, 0] @ r2["k_rot"][0, 1, 0]
    assert abs(s1 - s2) < 1e-9
    r3 = _append_case(oracle_mod, np.array([[100, 95]], np.int32), D=D, hq=2, hkv=2, seed=4)
    assert abs(r3["q_rot"][0, 0, 0] @ r3["k_rot"][0, 1, 0] - s1) > 1e-6


def test_rope_frequency_endpoints(oracle_mod):
    """Pair 0 rotates by pos radians; the last pair by pos * base^(-(D-2)/D)."""
    pos = np.array([[12345]], np.int32)
    r = _append_case(oracle_mod, pos, D=128, hq=1, hkv=1)
    x = brute.bits_to_f64(r["qb"])[0, 0, 0]
    y = r["q_rot"][0, 0, 0]
    assert abs(y[0] - (x[0] * math.cos(12345.0) - x[64] * math.sin(12345.0))) < 1e-12
    t = 12345.0 * 10.0 ** (-6.0 * 126.0 / 128.0)
    assert abs(y[127] - (x[127] * math.cos(t) + x[63] * math.sin(t))) < 1e-12


def test_append_writes_slots_and_rounds_to_nearest_even(oracle_mod):
    pos = np.array([[7, 8], [9, 10]], np.int32)
    r = _append_case(oracle_mod, pos, D=128, hq=4, hkv=2, n0=3)
    n0, n_new = r["n0"], r["n_new"]
    untouched = np.full(128, 0x40E0, np.uint16)  # bf16 7.0 fill
    for c in range(2):
        for h in range(2):
            for m in range(r["dk"].shape[2]):
                if n0 <= m < n0 + n_new:
                    i = m - n0
                    assert np.array_equal(r["dv"][c, h, m], r["vb"][c, i, h])
                    expect = np.array([oracle_mod.round_bf16(v) for v in r["k_rot"][c, i, h]], np.uint16)
                    assert np.array_equal(r["dk"][c, h, m], expect)
                else:
                    assert np.array_equal(r["dk"][c, h, m], untouched)
                    assert np.array_equal(r["dv"][c, h, m], untouched)
    rounded = torch.from_numpy(r["q_rot"]).to(torch.float32).to(torch.bfloat16)
    # Single rounding float32 -> bf16 agrees with direct rounding except where float32 rounding created a tie.
    same = (wl.bf16_bits(rounded) == r["q_out"]).mean()
    assert same > 0.999


def test_round_bf16_matches_float32_path_on_float_values(oracle_mod):
    rng = np.random.default_rng(0)
    vals = np.concatenate([rng.standard_normal(2000).astype(np.float32),
                           (rng.standard_normal(500) * 1e-38).astype(np.float32),
                           np.array([0.0, -0.0, 1.0, 65504.0, 3.0e38, -3.4e38, 1e-45], np.float32)])
    # exact ties: bf16 value + half ulp
    base = np.array([1.0, 1.5, -2.0, 3.0e-3], np.float32)
    ties = [np.nextafter(b, np.float32(np.inf)) for b in base]
    vals = np.concatenate([vals, base * np.float32(1 + 2 ** -8), base * np.float32(1 + 3 * 2 ** -8),
                           np.array(ties, np.float32)])
    ref = wl.bf16_bits(torch.from_numpy(vals).to(torch.bfloat16))
    got = np.array([oracle_mod.round_bf16(float(v)) for v in vals], np.uint16)
    assert np.array_equal(got, ref)


def test_round_bf16_no_double_rounding(oracle_mod):
    # x = 1 + 2^-8 + 2^-30: just above the tie between bf16 1.0 and 1.0078125 -> rounds up.
    # Rounding to float32 first would give exactly the tie 1 + 2^-8 and then round to even (down).
    x = 1.0 + 2.0 ** -8 + 2.0 ** -30
    assert oracle_mod.round_bf16(x) == 0x3F81
    assert oracle_mod.round_bf16(1.0 + 2.0 ** -8) == 0x3F80            # tie -> even
    assert oracle_mod.round_bf16(1.0 + 3 * 2.0 ** -8) == 0x3F82        # tie -> even (up)
    assert oracle_mod.round_bf16(-(1.0 + 2.0 ** -8 + 2.0 ** -40)) == 0xBF81
    assert oracle_mod.round_bf16(float("inf")) == 0x7F80
    assert oracle_mod.round_bf16(3.4e38) == 0x7F80                       # above bf16 max -> inf
