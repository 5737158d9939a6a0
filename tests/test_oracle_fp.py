"""Pins of the oracle's non-finite count and fp64 sum of squares.

* closed forms: constant tensors give exactly n*c^2;
* the exact rational sum of squares (fractions.Fraction) and the correctly
  rounded sum (math.fsum) on small random inputs, within the fp64 bound of a
  sequential sum of n non-negative terms, (n-1) * 2^-53 relative;
* bf16 decoding against torch's own bf16 -> fp32 conversion;
* the non-finite count equals the count of injected NaN/Inf positions and
  those elements are excluded from the sum.
"""
import math
import random
import struct
from fractions import Fraction

import numpy as np
import pytest
import torch

DT_BYTES, DT_BF16, DT_F32 = 0, 1, 2
U = 2.0 ** -53


def _f32_bytes(vals):
    return np.asarray(vals, dtype=np.float32).tobytes()


def test_constant_f32_closed_form(orc):
    for c, n in [(0.5, 1000), (3.0, 4097), (0.0, 10), (-2.0, 513)]:
        nf, s = orc.fp_values(_f32_bytes([c] * n), DT_F32)
        assert nf == 0
        assert s == n * c * c


def test_constant_bf16_closed_form(orc):
    t = torch.full((777,), 0.25, dtype=torch.bfloat16)
    nf, s = orc.fp_values(t.view(torch.uint8).numpy().tobytes(), DT_BF16)
    assert nf == 0 and s == 777 * 0.0625


def _rand_f32(rng, n):
    out = []
    for _ in range(n):
        e = rng.randrange(-40, 40)
        out.append(rng.uniform(-1, 1) * 2.0 ** e)
    return np.asarray(out, dtype=np.float32)


def test_exact_rational_and_fsum(orc):
    rng = random.Random(11)
    for n in [1, 2, 5, 33, 256, 1000]:
        x = _rand_f32(rng, n)
        exact = sum(Fraction(float(v)) ** 2 for v in x)
        nf, s = orc.fp_values(x.tobytes(), DT_F32)
        assert nf == 0
        bound = max(n - 1, 1) * U * float(exact)
        assert abs(Fraction(s) - exact) <= Fraction(bound)
        fs = math.fsum(float(v) * float(v) for v in x)  # each square is exact in fp64
        assert abs(s - fs) <= bound


def test_subnormal_and_huge_values(orc):
    x = np.array([1e-45, -3e-42, 1e-38, 3e38, -1.7e38, 0.0, -0.0], dtype=np.float32)
    exact = sum(Fraction(float(v)) ** 2 for v in x)
    nf, s = orc.fp_values(x.tobytes(), DT_F32)
    assert nf == 0
    assert abs(Fraction(s) - exact) <= Fraction(6 * U * float(exact))


def test_nonfinite_counted_and_excluded(orc):
    rng = random.Random(12)
    x = _rand_f32(rng, 2000)
    pos = sorted(rng.sample(range(2000), 37))
    specials = [float("nan"), float("inf"), float("-inf")]
    for i, p in enumerate(pos):
        x[p] = specials[i % 3]
    # a NaN with a payload and a negative NaN are still non-finite
    raw = bytearray(x.tobytes())
    raw[4 * pos[0]: 4 * pos[0] + 4] = struct.pack("<I", 0xFFC12345)
    nf, s = orc.fp_values(bytes(raw), DT_F32)
    assert nf == len(pos)
    keep = [float(v) for i, v in enumerate(x) if i not in set(pos)]
    assert abs(s - math.fsum(v * v for v in keep)) <= len(keep) * U * s


def test_bf16_decoding_matches_torch(orc):
    rng = random.Random(13)
    bits = []
    while len(bits) < 500:
        b = rng.getrandbits(16)
        if (b & 0x7F80) != 0x7F80:
            bits.append(b)
    raw = np.asarray(bits, dtype=np.uint16)
    vals = torch.from_numpy(raw.view(np.int16).copy()).view(torch.bfloat16).to(torch.float32)
    for i in range(0, 500, 50):
        nf, s = orc.fp_values(raw[i:i + 1].tobytes(), DT_BF16)
        assert nf == 0
        assert s == float(vals[i]) ** 2
    nf, s = orc.fp_values(raw.tobytes(), DT_BF16)
    assert abs(s - math.fsum(float(v) ** 2 for v in vals)) <= 500 * U * s


def test_bf16_nonfinite(orc):
    raw = np.array([0x3F80, 0x7F80, 0xFF80, 0x7FC0, 0xFFC1, 0x4000], dtype=np.uint16)
    nf, s = orc.fp_values(raw.tobytes(), DT_BF16)
    assert nf == 4 and s == 1.0 + 4.0


def test_bytes_dtype_has_no_values(orc):
    nf, s = orc.fp_values(bytes(range(256)) * 3, DT_BYTES)
    assert nf == 0 and s == 0.0


def test_weight_and_master_agree(orc):
    """The generator makes master == float(bf16 weight); their sums agree."""
    from paper_2509_03047_gb300 import synth

    cfg = synth.get_config("tiny")
    state = synth.make_state(cfg, "cpu")
    for t in range(0, 8, 3):
        w, m = state[4 * t], state[4 * t + 1]
        _, sw = orc.fp_values(w.view(torch.uint8).numpy().tobytes(), DT_BF16)
        _, sm = orc.fp_values(m.view(torch.uint8).numpy().tobytes(), DT_F32)
        assert sw == sm


def test_fingerprint_chunk_uses_crc32c(orc):
    data = _f32_bytes([1.0, 2.0, float("nan")])
    crc, nf, s = orc.fingerprint_chunk(data, DT_F32)
    assert crc == orc.crc32c(data) and nf == 1 and s == 5.0
