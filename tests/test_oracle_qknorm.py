"""Pins for the oracle's QK-norm append (App. D, Tab. ablations, "QK-Norm" regime); no GPU.

The answers come from outside the oracle's own formula: the unit RMS of every
normalised head (RoPE keeps each pair's norm), invariance to the head's
scale, a constant head's closed form, one-hot weights that expose where the
weights act (before RoPE: the weight of dimension j shows up in j's rotation
partner), a head's independence from the others, RoPE as a complex
multiplication at a hand-computed angle, and hand-placed draft slots.  The
planted mistakes in tests/test_oracle_qknorm_mutations.py each fail one of them.
"""
import importlib.util
import os

import numpy as np
import pytest

if os.environ.get("KVO_QKNORM_OVERRIDE"):  # a copy with a planted mistake
    _spec = importlib.util.spec_from_file_location("oracle.qknorm_under_test", os.environ["KVO_QKNORM_OVERRIDE"])
    import oracle  # noqa: F401  (the package, for the copy's relative imports)
    qo = importlib.util.module_from_spec(_spec)
    qo.__package__ = "oracle"
    _spec.loader.exec_module(qo)
else:
    from oracle import qknorm as qo

D = 128
ONES = np.full(D, 0x3F80, dtype=np.uint16)  # bf16 1.0


def _bits(x):
    """fp32 values exactly representable in bf16 -> bit patterns."""
    return (np.asarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


def _bf16_round(rng, shape, scale=1.0):
    x = (rng.standard_normal(shape) * scale).astype(np.float32)
    return _bits(x.view(np.uint32) & 0xFFFF0000)


def _inputs(rng, C=2, n=3, hq=4, hkv=2, scale=1.0):
    return (_bf16_round(rng, (C, n, hq, D), scale), _bf16_round(rng, (C, n, hkv, D), scale),
            _bf16_round(rng, (C, n, hkv, D), scale))


def test_unit_rms_after_norm_and_rope():
    rng = np.random.default_rng(1)
    q, k, v = _inputs(rng, scale=7.0)
    pos = rng.integers(0, 50000, (2, 3))
    qn, kn, _ = qo.append_qknorm(q, k, v, pos, 0, 1e6, ONES, ONES, 1e-12, 3)
    np.testing.assert_allclose(np.sqrt(np.mean(qn * qn, axis=-1)), 1.0, rtol=1e-9)
    np.testing.assert_allclose(np.sqrt(np.mean(kn * kn, axis=-1)), 1.0, rtol=1e-9)


def test_invariant_to_the_head_scale():
    rng = np.random.default_rng(2)
    x = rng.standard_normal((5, D))
    w = rng.standard_normal(D)
    np.testing.assert_allclose(qo.rms_norm(1024.0 * x, w, 1e-12), qo.rms_norm(x, w, 1e-12), rtol=1e-9, atol=1e-12)


def test_constant_head_closed_form():
    # x_j = c for every j: mean square c^2, so RMSNorm(x) = c / sqrt(c^2 + eps) * w.
    w = np.linspace(-2, 3, D)
    for c, eps in ((0.5, 0.25), (-3.0, 1e-6), (0.01, 1e-2)):
        got = qo.rms_norm(np.full((1, D), c), w, eps)
        np.testing.assert_allclose(got[0], c / np.sqrt(c * c + eps) * w, rtol=1e-13)


def test_zero_head_stays_zero():
    got = qo.rms_norm(np.zeros((2, D)), np.ones(D), 1e-6)
    assert np.array_equal(got, np.zeros((2, D)))


def test_one_hot_weight_acts_before_rope():
    # w = e_j (j < 64): after the norm only dimension j is left, x_j / rms; RoPE then moves it to the
    # pair (j, j + 64) as (cos theta_j, sin theta_j) times that value, theta_j = pos * base^(-2j/128).
    rng = np.random.default_rng(3)
    x = _bf16_round(rng, (1, 1, 1, D))
    xf = x.astype(np.uint32) << 16
    xf = xf.view(np.float32).astype(np.float64)[0, 0, 0]
    rms = np.sqrt(np.mean(xf * xf) + 1e-6)
    base, p = 10000.0, 37
    for j in (0, 5, 63):
        w = np.zeros(D, dtype=np.float32)
        w[j] = 1.0
        qn, _, _ = qo.append_qknorm(x, x[:, :, :1], x[:, :, :1], np.array([[p]]), 0, base, _bits(w), ONES, 1e-6, 1)
        theta = p * base ** (-2.0 * j / D)
        expect = np.zeros(D)
        expect[j] = xf[j] / rms * np.cos(theta)
        expect[j + 64] = xf[j] / rms * np.sin(theta)
        np.testing.assert_allclose(qn[0, 0, 0], expect, rtol=1e-12, atol=1e-15)


def test_heads_are_normalised_separately():
    rng = np.random.default_rng(4)
    q, k, v = _inputs(rng, C=1, n=1, hq=3, hkv=1)
    pos = np.array([[11]])
    a, _, _ = qo.append_qknorm(q, k, v, pos, 0, 1e6, ONES, ONES, 1e-6, 1)
    q2 = q.copy()
    q2[0, 0, 1] = _bits(np.linspace(-50, 50, D).astype(np.float32).view(np.uint32) & 0xFFFF0000)
    b, _, _ = qo.append_qknorm(q2, k, v, pos, 0, 1e6, ONES, ONES, 1e-6, 1)
    assert np.array_equal(a[0, 0, 0], b[0, 0, 0]) and np.array_equal(a[0, 0, 2], b[0, 0, 2])
    assert not np.allclose(a[0, 0, 1], b[0, 0, 1])


def test_rope_as_complex_rotation_with_distinct_q_and_k_weights():
    rng = np.random.default_rng(5)
    q, k, v = _inputs(rng, C=1, n=2, hq=2, hkv=1)
    wq, wk = _bf16_round(rng, D), _bf16_round(rng, D)
    pos = np.array([[3, 900]])
    base, eps = 5e5, 1e-6
    qn, kn, _ = qo.append_qknorm(q, k, v, pos, 0, base, wq, wk, eps, 2)

    def widen(b):
        return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)

    for x, w, got in ((widen(q)[0, :, 1], widen(wq), qn[0, :, 1]), (widen(k)[0, :, 0], widen(wk), kn[0, 0])):
        for i in range(2):
            y = x[i] / np.sqrt(np.mean(x[i] ** 2) + eps) * w
            z = (y[:64] + 1j * y[64:]) * np.exp(1j * pos[0, i] * base ** (-np.arange(64) / 64.0))
            np.testing.assert_allclose(got[i], np.concatenate([z.real, z.imag]), rtol=1e-11, atol=1e-13)


def test_values_unchanged_and_slots_by_hand():
    rng = np.random.default_rng(6)
    C, n, hkv = 2, 3, 2
    q, k, v = _inputs(rng, C=C, n=n, hkv=hkv)
    _, kn, vs = qo.append_qknorm(q, k, v, np.zeros((C, n), dtype=np.int64), 4, 1e6, ONES, ONES, 1e-6, 8)
    vf = (v.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    for c in range(C):
        for h in range(hkv):
            for i in range(n):
                assert np.array_equal(vs[c, h, i], vf[c, i, h])  # slot n0 + i of (c, h) holds node i's value
    assert kn.shape == (C, hkv, n, D)


def test_arguments_are_checked():
    rng = np.random.default_rng(7)
    q, k, v = _inputs(rng)
    pos = np.zeros((2, 3), dtype=np.int64)
    with pytest.raises(ValueError):
        qo.append_qknorm(q, k, v, pos, 0, 1e6, ONES, ONES, 0.0, 3)
    with pytest.raises(ValueError):
        qo.append_qknorm(q, k, v, pos, 1, 1e6, ONES, ONES, 1e-6, 3)
    with pytest.raises(ValueError):
        qo.rms_norm(np.zeros((2, 64)), np.ones(64), 1e-6)
