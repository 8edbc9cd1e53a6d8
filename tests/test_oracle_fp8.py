"""Pins for the oracle's e4m3 decoding of the fp8 target cache; no GPU.

The answers come from outside the oracle's formula: PyTorch's float8_e4m3fn
decoding of all 256 codes (an independent implementation), values fixed by
the format (zero, signed zero, the smallest subnormal, the largest subnormal,
the smallest normal, one, the largest finite value, NaN), monotonic order of
the non-negative codes, and the exact bf16 round trip at extreme scales.  The
planted mistakes in tests/test_oracle_fp8_mutations.py each fail one of them.
"""
import importlib.util
import os

import numpy as np
import pytest

if os.environ.get("KVO_FP8_OVERRIDE"):  # a copy with a planted mistake
    _spec = importlib.util.spec_from_file_location("fp8_under_test", os.environ["KVO_FP8_OVERRIDE"])
    fo = importlib.util.module_from_spec(_spec)
    _spec.loader.exec_module(fo)
else:
    from oracle import fp8 as fo

ALL = np.arange(256, dtype=np.uint8)


def test_matches_torch_float8_e4m3fn_on_every_code():
    torch = pytest.importorskip("torch")
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("torch without float8_e4m3fn")
    ref = torch.from_numpy(ALL.copy()).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    got = fo.e4m3_value(ALL)
    assert np.array_equal(np.isnan(got), np.isnan(ref))
    ok = ~np.isnan(ref)
    assert np.array_equal(got[ok], ref[ok])


@pytest.mark.parametrize("code,value", [
    (0x00, 0.0), (0x01, 2.0 ** -9), (0x07, 7 * 2.0 ** -9), (0x08, 2.0 ** -6), (0x38, 1.0), (0x39, 1.125),
    (0x40, 2.0), (0x7E, 448.0), (0xFE, -448.0), (0xB8, -1.0), (0x81, -(2.0 ** -9)),
])
def test_values_fixed_by_the_format(code, value):
    assert fo.e4m3_value(np.array([code], dtype=np.uint8))[0] == value


def test_signed_zero_and_nan_codes():
    v = fo.e4m3_value(np.array([0x80, 0x7F, 0xFF, 0x7E, 0x77], dtype=np.uint8))
    assert v[0] == 0.0 and np.signbit(v[0])
    assert np.isnan(v[1]) and np.isnan(v[2])
    assert not np.isnan(v[3]) and not np.isnan(v[4])  # e = 15 with m < 7 is finite


def test_non_negative_codes_increase():
    v = fo.e4m3_value(ALL[:0x7F])
    assert np.all(np.diff(v) > 0)
    assert np.array_equal(fo.e4m3_value(ALL[0x80:0xFF]), -v)


@pytest.mark.parametrize("exp", [-64, -3, 0, 5, 64])
def test_bf16_bits_are_the_exact_scaled_value(exp):
    bits = fo.dequant_bf16_bits(ALL, exp)
    widened = (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    v = fo.e4m3_value(ALL) * 2.0 ** exp
    ok = ~np.isnan(v)
    assert np.array_equal(widened[ok], v[ok])
    assert np.all(bits[~ok] == fo.BF16_NAN)


def test_quantisation_error_of_an_fp8_cache():
    """The tolerance study of the fp8 variant (not a pin of the decoder): the same attention on a
    bf16 cache and on its e4m3 codes (scales 2^-3, 2^-2; round to nearest) differs by ~2.7% rel-L2 in
    the output and ~1e-4 in lse for N(0, 1) keys and values -- the error of e4m3's 3-bit mantissa,
    ten times the bf16 path's parity tolerance, so an fp8 cache is a drafter-quality trade-off."""
    if os.environ.get("KVO_FP8_OVERRIDE"):
        pytest.skip("pins only")
    torch = pytest.importorskip("torch")
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("torch without float8_e4m3fn")
    from paper_2604_26412_gb300 import workloads as wl
    from tests import gpu_helpers as gh
    spec = wl.Spec("study", 1, 1, [2048], [4, 4], True, True, page_size=16, hq=32, hkv=8, seed=5)
    inp = wl.make_inputs(spec, "cpu", seed=5)
    N, Nq = spec.n_nodes, 4
    dk, dv = wl.random_draft_kv(spec, inp.n_max, N, "cpu", seed=6)
    q = wl.random_queries(spec, Nq, "cpu", seed=7)
    ob, lb = gh.oracle_attn(gh.HostCache(inp), q, dk, dv, N, Nq)
    tk8, tv8 = wl.fp8_target(inp)
    hf = gh.HostCache(inp)
    hf.tk = fo.dequant_bf16_bits(tk8.numpy(), wl.FP8_K_EXP)
    hf.tv = fo.dequant_bf16_bits(tv8.numpy(), wl.FP8_V_EXP)
    of, lf = gh.oracle_attn(hf, q, dk, dv, N, Nq)
    rel = np.linalg.norm(of - ob) / np.linalg.norm(ob)
    assert 0.01 < rel < 0.06, rel
    assert np.abs(lf - lb).max() < 1e-3
