"""CPU oracle for the fp8 target cache: exact decoding of e4m3 codes -- numpy.

TEST INFRASTRUCTURE ONLY.  Only tests, the package's ``smoke()`` self-check and
``bench.py``'s CPU-baseline leg may import it; the library never does, and
nothing here imports the library.

Not from the paper: an fp8 KV cache is a compression variant of the target
cache (the hot path's KVSHOT_TARGET_FP8 flag).  Definition (OCP 8-bit floating
point, format E4M3): bit 7 is the sign, bits 6..3 the exponent e with bias 7,
bits 2..0 the mantissa m; e > 0 encodes (1 + m/8) 2^(e-7), e = 0 encodes the
subnormal (m/8) 2^-6; the two codes with e = 15 and m = 7 are NaN and there are
no infinities (so the largest magnitude is 1.75 x 2^8 = 448).  A cached key or
value is the decoded code times 2^exp for the cache's scale exponent, which is
exact in bf16: at most 4 significant bits, exponents well inside bf16's range.
The attention oracle then runs on those bf16 values unchanged.
"""
from __future__ import annotations

import numpy as np

BF16_NAN = 0x7FC0


def e4m3_value(codes) -> np.ndarray:
    """Decoded fp64 values of uint8 e4m3 codes (NaN for the two NaN codes)."""
    c = np.asarray(codes, dtype=np.uint8).astype(np.int64)
    sign = np.where((c >> 7) & 1, -1.0, 1.0)
    e = (c >> 3) & 0xF
    m = (c & 7).astype(np.float64)
    mag = np.where(e > 0, (1.0 + m / 8.0) * np.exp2(e - 7.0), (m / 8.0) * 2.0 ** -6)
    val = sign * mag
    return np.where((e == 15) & ((c & 7) == 7), np.nan, val)


def dequant_bf16_bits(codes, scale_exp: int) -> np.ndarray:
    """bf16 bit patterns (uint16) of e4m3(code) * 2^scale_exp; NaN codes give the canonical NaN."""
    v = e4m3_value(codes) * 2.0 ** int(scale_exp)
    f = v.astype(np.float32)  # exact: at most 4 significant bits
    bits = (f.view(np.uint32) >> 16).astype(np.uint16)
    return np.where(np.isnan(v), np.uint16(BF16_NAN), bits)
