"""Pins for the oracle's gated-delta fusion (Sec. 3.4, Eqs. "delta" and "fusion"); no GPU.

Each case fixes the answer by something other than the oracle's own formula:
a special case whose result the equations force (no correction, a closed or
open gate, g = 1/2), scipy's logistic function, a one-hot probe that reads one
column of a weight matrix back, or a symmetry (linearity in W_delta).  A block
of W_g taken in the wrong order, a transposed weight matrix, a dropped bias, a
sign flip in delta or a missing n in the residual each fail at least one.
"""
import importlib.util
import os

import numpy as np
import pytest
from scipy.special import expit

if os.environ.get("KVO_FUSION_OVERRIDE"):  # a copy with a planted mistake (tests/test_oracle_fusion_mutations.py)
    _spec = importlib.util.spec_from_file_location("fusion_under_test", os.environ["KVO_FUSION_OVERRIDE"])
    fo = importlib.util.module_from_spec(_spec)
    _spec.loader.exec_module(fo)
else:
    from oracle import fusion as fo


def _rand(rng, T, d, scale_w=None):
    n = rng.standard_normal((T, d))
    o = rng.standard_normal((T, d))
    sw = scale_w if scale_w is not None else 1.0 / np.sqrt(3 * d)
    w_g = rng.standard_normal((d, 3 * d)) * sw
    b_g = rng.standard_normal(d) * 0.3
    w_d = rng.standard_normal((d, d)) / np.sqrt(d)
    return n, o, w_g, b_g, w_d


def test_no_correction_when_branches_agree():
    # o = n: delta = 0, so h = n whatever the weights (the drafter falls back to the EAGLE-3 path).
    rng = np.random.default_rng(1)
    n, _, w_g, b_g, w_d = _rand(rng, 5, 12)
    h = fo.gated_delta(n, n.copy(), w_g, b_g, w_d)
    assert np.array_equal(h, n)


def test_closed_gate_keeps_the_self_attention_branch():
    # W_g = 0 and b_g very negative: g ~ 0, h = n (Sec. 3.4: "the model reduces to standard EAGLE-3").
    rng = np.random.default_rng(2)
    n, o, _, _, w_d = _rand(rng, 4, 8)
    d = n.shape[1]
    h = fo.gated_delta(n, o, np.zeros((d, 3 * d)), np.full(d, -60.0), w_d)
    np.testing.assert_allclose(h, n, rtol=0, atol=1e-20)


def test_open_gate_with_identity_projection_gives_the_cross_branch():
    # W_g = 0, b_g very positive (g ~ 1) and W_delta = I: h = n + (o - n) = o.
    rng = np.random.default_rng(3)
    n, o, _, _, _ = _rand(rng, 3, 8)
    d = n.shape[1]
    h = fo.gated_delta(n, o, np.zeros((d, 3 * d)), np.full(d, 60.0), np.eye(d))
    np.testing.assert_allclose(h, o, rtol=0, atol=1e-12)


def test_half_open_gate():
    # W_g = 0, b_g = 0: g = 1/2 exactly, h = n + (o - n) W_delta^T / 2.
    rng = np.random.default_rng(4)
    n, o, _, _, w_d = _rand(rng, 6, 10)
    d = n.shape[1]
    h = fo.gated_delta(n, o, np.zeros((d, 3 * d)), np.zeros(d), w_d)
    expect = n + 0.5 * np.einsum("ij,tj->ti", w_d, o - n)
    np.testing.assert_allclose(h, expect, rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("block", [0, 1, 2])
def test_gate_reads_the_right_input_block(block):
    # W_g = [I 0 0], [0 I 0] or [0 0 I]: the gate's pre-activation is n, o or delta = o - n; with
    # W_delta = I the output is n + expit(that) * (o - n).
    rng = np.random.default_rng(10 + block)
    n, o, _, _, _ = _rand(rng, 4, 6)
    d = n.shape[1]
    w_g = np.zeros((d, 3 * d))
    w_g[:, block * d:(block + 1) * d] = np.eye(d)
    h = fo.gated_delta(n, o, w_g, np.zeros(d), np.eye(d))
    pre = (n, o, o - n)[block]
    np.testing.assert_allclose(h, n + expit(pre) * (o - n), rtol=1e-13, atol=1e-13)


def test_bias_sets_the_gate_when_the_weights_vanish():
    rng = np.random.default_rng(5)
    n, o, _, _, _ = _rand(rng, 3, 5)
    d = n.shape[1]
    beta = np.array([-3.0, -0.5, 0.0, 0.75, 4.0])
    h = fo.gated_delta(n, o, np.zeros((d, 3 * d)), beta, np.eye(d))
    np.testing.assert_allclose(h, n + expit(beta) * (o - n), rtol=1e-13, atol=1e-13)


def test_one_hot_delta_reads_a_column_of_w_delta():
    # n = 0, o = e_j (so delta = e_j), open gate: h = W_delta e_j, the j-th column (not the row).
    rng = np.random.default_rng(6)
    d = 7
    w_d = rng.standard_normal((d, d))
    for j in (0, 3, 6):
        o = np.zeros((1, d))
        o[0, j] = 1.0
        h = fo.gated_delta(np.zeros((1, d)), o, np.zeros((d, 3 * d)), np.full(d, 60.0), w_d)
        np.testing.assert_allclose(h[0], w_d[:, j], rtol=0, atol=1e-12)


def test_one_hot_input_reads_a_column_of_w_g():
    # n = 0, o = e_j: the gate's pre-activation is W_g's columns d + j and 2d + j summed (o and delta both e_j).
    rng = np.random.default_rng(7)
    d = 5
    w_g = rng.standard_normal((d, 3 * d))
    for j in (1, 4):
        o = np.zeros((1, d))
        o[0, j] = 1.0
        h = fo.gated_delta(np.zeros((1, d)), o, w_g, np.zeros(d), np.eye(d))
        g = expit(w_g[:, d + j] + w_g[:, 2 * d + j])
        np.testing.assert_allclose(h[0], g * o[0], rtol=1e-13, atol=1e-13)


def test_linear_in_w_delta_at_fixed_gate():
    rng = np.random.default_rng(8)
    n, o, w_g, b_g, w_a = _rand(rng, 5, 9)
    w_b = rng.standard_normal(w_a.shape)
    ha = fo.gated_delta(n, o, w_g, b_g, w_a) - n
    hb = fo.gated_delta(n, o, w_g, b_g, w_b) - n
    hab = fo.gated_delta(n, o, w_g, b_g, w_a + w_b) - n
    np.testing.assert_allclose(hab, ha + hb, rtol=1e-12, atol=1e-12)


def test_sigmoid_matches_scipy_over_a_wide_range():
    z = np.linspace(-700, 700, 2001)
    np.testing.assert_allclose(fo.sigmoid(z), expit(z), rtol=1e-15, atol=0)
    np.testing.assert_array_equal(fo.sigmoid(np.array([-1e6, 0.0, 1e6])), [0.0, 0.5, 1.0])


def test_bf16_bit_patterns_are_widened_exactly():
    bits = np.array([0x3F80, 0xC000, 0x3E80, 0x0000, 0x8000, 0x7F7F], dtype=np.uint16)
    np.testing.assert_array_equal(fo.widen(bits), [1.0, -2.0, 0.25, 0.0, -0.0, 3.3895313892515355e38])


def test_shapes_are_checked():
    with pytest.raises(ValueError):
        fo.gated_delta(np.zeros((2, 4)), np.zeros((2, 4)), np.zeros((4, 8)), np.zeros(4), np.zeros((4, 4)))
