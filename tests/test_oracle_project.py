"""Pins for the oracle's multi-layer KV projection and RoPE fix (Sec. 3.2); no GPU.

The answers come from outside the oracle's own formula: a selector matrix
that reads one layer back, RoPE at position 0 (identity), RoPE as a complex
multiplication (an independent formulation), the norm of every rotated pair,
the composition of two rotations, and hand-computed cache rows.  The planted
mistakes in tests/test_oracle_project_mutations.py each fail one of them.
"""
import importlib.util
import os

import numpy as np
import pytest

if os.environ.get("KVO_PROJECT_OVERRIDE"):  # a copy with a planted mistake
    _spec = importlib.util.spec_from_file_location("oracle.project_under_test", os.environ["KVO_PROJECT_OVERRIDE"],
                                                   submodule_search_locations=None)
    import oracle  # noqa: F401  (the package, for the copy's relative import)
    po = importlib.util.module_from_spec(_spec)
    po.__package__ = "oracle"
    _spec.loader.exec_module(po)
else:
    from oracle import project as po

D = 128


def _inputs(rng, T, L, hkv):
    k = rng.standard_normal((T, L, hkv, D))
    v = rng.standard_normal((T, L, hkv, D))
    return k, v


def _selector(L, hkv, layer):
    dkv = hkv * D
    w = np.zeros((dkv, L * dkv))
    w[:, layer * dkv:(layer + 1) * dkv] = np.eye(dkv)
    return w


@pytest.mark.parametrize("layer", [0, 1, 2])
def test_selector_reads_one_layer_back(layer):
    rng = np.random.default_rng(layer)
    T, L, hkv = 4, 3, 2
    k, v = _inputs(rng, T, L, hkv)
    w = _selector(L, hkv, layer)
    kp, vp = po.kv_project(k, v, w, w, np.arange(T) * 7, 1e6, apply_rope=False)
    np.testing.assert_array_equal(kp, k[:, layer].reshape(T, -1))
    np.testing.assert_array_equal(vp, v[:, layer].reshape(T, -1))


def test_rope_at_position_zero_is_the_identity():
    rng = np.random.default_rng(5)
    k, v = _inputs(rng, 3, 2, 2)
    w = _selector(2, 2, 1)
    kp, _ = po.kv_project(k, v, w, w, np.zeros(3, dtype=np.int64), 1e6, apply_rope=True)
    np.testing.assert_allclose(kp, k[:, 1].reshape(3, -1), rtol=0, atol=1e-15)


def test_rope_matches_complex_rotation():
    # Each head's pair (x_j, x_{j+64}) is the complex number x_j + i x_{j+64} times e^{i theta_j}.
    rng = np.random.default_rng(6)
    T, hkv, base = 5, 3, 1.0e6
    x = rng.standard_normal((T, hkv * D))
    pos = np.array([0, 1, 17, 4095, 32767])
    got = po.rope(x, pos, base)
    z = x.reshape(T, hkv, D)[..., :64] + 1j * x.reshape(T, hkv, D)[..., 64:]
    theta = pos[:, None, None] * np.power(base, -np.arange(64) / 64.0)[None, None, :]
    r = z * np.exp(1j * theta)
    want = np.concatenate([r.real, r.imag], axis=-1).reshape(T, -1)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


def test_rope_keeps_every_pair_norm_and_composes():
    rng = np.random.default_rng(7)
    x = rng.standard_normal((4, 2 * D))
    p1, p2 = np.array([3, 100, 2000, 9]), np.array([5, 7, 11, 30000])
    y = po.rope(x, p1, 1e4)
    n0 = np.hypot(x.reshape(4, 2, D)[..., :64], x.reshape(4, 2, D)[..., 64:])
    n1 = np.hypot(y.reshape(4, 2, D)[..., :64], y.reshape(4, 2, D)[..., 64:])
    np.testing.assert_allclose(n1, n0, rtol=1e-13)
    np.testing.assert_allclose(po.rope(y, p2, 1e4), po.rope(x, p1 + p2, 1e4), rtol=1e-9, atol=1e-9)


def test_values_ignore_positions_and_rope():
    rng = np.random.default_rng(8)
    T, L, hkv = 3, 2, 1
    k, v = _inputs(rng, T, L, hkv)
    wk = rng.standard_normal((hkv * D, L * hkv * D))
    wv = rng.standard_normal((hkv * D, L * hkv * D))
    _, v1 = po.kv_project(k, v, wk, wv, np.array([0, 1, 2]), 1e6, apply_rope=True)
    _, v2 = po.kv_project(k, v, wk, wv, np.array([9, 99, 999]), 1e6, apply_rope=False)
    np.testing.assert_array_equal(v1, v2)


def test_linear_in_the_weights():
    rng = np.random.default_rng(9)
    T, L, hkv = 4, 3, 1
    k, v = _inputs(rng, T, L, hkv)
    wa, wb = (rng.standard_normal((hkv * D, L * hkv * D)) for _ in range(2))
    pos = np.array([1, 2, 3, 4])
    ka, _ = po.kv_project(k, v, wa, wa, pos, 1e6, True)
    kb, _ = po.kv_project(k, v, wb, wb, pos, 1e6, True)
    kab, _ = po.kv_project(k, v, wa + wb, wa + wb, pos, 1e6, True)
    np.testing.assert_allclose(kab, ka + kb, rtol=1e-10, atol=1e-10)


def test_cache_rows_by_hand():
    # Paged: cache 0's pages are [3, 1]; page size 4, hkv 2.  Position 5 -> page 1 (pool page 1), slot 1.
    pt = np.array([[3, 1], [0, 2]])
    rows = po.cache_rows([0, 1, 0], [5, 2, 0], 2, page_table=pt, page_size=4)
    np.testing.assert_array_equal(rows, [[(1 * 2 + 0) * 4 + 1, (1 * 2 + 1) * 4 + 1],
                                         [(0 * 2 + 0) * 4 + 2, (0 * 2 + 1) * 4 + 2],
                                         [(3 * 2 + 0) * 4 + 0, (3 * 2 + 1) * 4 + 0]])
    # Contiguous: [C, hkv, l_cap] rows.
    np.testing.assert_array_equal(po.cache_rows([1], [3], 2, l_cap=10), [[(1 * 2 + 0) * 10 + 3, (1 * 2 + 1) * 10 + 3]])


def test_shapes_are_checked():
    with pytest.raises(ValueError):
        po.kv_project(np.zeros((1, 2, 1, D)), np.zeros((1, 2, 1, D)), np.zeros((D, D)), np.zeros((D, D)),
                      np.zeros(1), 1e6, True)
