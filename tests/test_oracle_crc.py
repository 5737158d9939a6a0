"""Pins of the oracle's CRC-32C against facts outside the oracle.

* the standard CRC-32C check value of "123456789" (tests/golden);
* zlib's independent CRC-32 (IEEE polynomial 0xEDB88320, same reflection,
  preset and final XOR) for the oracle's polynomial-generic table, bitwise and
  combine code -- only the polynomial constant differs from CRC-32C, and that
  constant is pinned by the check value;
* mathematical invariants: affine linearity, the constant residue of a
  message followed by its own CRC, detection of every single-bit error and
  of every burst of at most 32 bits.
"""
import os
import random
import zlib

import pytest

CRC32C = 0x82F63B78
IEEE = 0xEDB88320
F = 0xFFFFFFFF
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "crc32c_check.txt")


def _golden():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                msg, val = line.split()
                rows.append((msg.encode(), int(val, 16)))
    return rows


def _rand_bytes(rng, n):
    return bytes(rng.getrandbits(8) for _ in range(n))


def test_check_value_table_and_bitwise(orc):
    for msg, val in _golden():
        assert orc.crc32c(msg) == val
        assert orc.crc_table(CRC32C, F, F, msg) == val
        assert orc.crc_bitwise(CRC32C, F, F, msg) == val


def test_empty_message_is_zero(orc):
    assert orc.crc32c(b"") == 0
    assert orc.crc_bitwise(CRC32C, F, F, b"") == 0


def test_generic_table_and_bitwise_match_zlib_ieee(orc):
    rng = random.Random(1)
    lengths = list(range(0, 70)) + [255, 256, 257, 1000, 4096 + 3]
    for n in lengths:
        data = _rand_bytes(rng, n)
        want = zlib.crc32(data) & F
        assert orc.crc_table(IEEE, F, F, data) == want, n
        assert orc.crc_bitwise(IEEE, F, F, data) == want, n


def test_table_equals_bitwise_crc32c(orc):
    rng = random.Random(2)
    for _ in range(300):
        data = _rand_bytes(rng, rng.randrange(0, 97))
        assert orc.crc32c(data) == orc.crc_bitwise(CRC32C, F, F, data)


def test_combine_matches_zlib_concatenation_ieee(orc):
    rng = random.Random(3)
    for _ in range(200):
        a = _rand_bytes(rng, rng.randrange(0, 300))
        b = _rand_bytes(rng, rng.randrange(0, 300))
        got = orc.crc_combine(IEEE, zlib.crc32(a) & F, zlib.crc32(b) & F, len(b))
        assert got == zlib.crc32(a + b) & F


def test_combine_identity_random_splits_crc32c(orc):
    rng = random.Random(4)
    for _ in range(300):
        m = _rand_bytes(rng, rng.randrange(0, 600))
        cut = rng.randrange(0, len(m) + 1)
        a, b = m[:cut], m[cut:]
        assert orc.crc32c_combine(orc.crc32c(a), orc.crc32c(b), len(b)) == orc.crc32c(m)


def test_affine_linearity(orc):
    """crc(a^b) ^ crc(a) ^ crc(b) == crc(0...0) for equal lengths."""
    rng = random.Random(5)
    for n in [1, 3, 4, 16, 61, 512]:
        for _ in range(20):
            a, b = _rand_bytes(rng, n), _rand_bytes(rng, n)
            x = bytes(i ^ j for i, j in zip(a, b))
            assert orc.crc32c(x) ^ orc.crc32c(a) ^ orc.crc32c(b) == orc.crc32c(bytes(n))


def test_residue_is_constant(orc):
    """Appending a message's CRC (little-endian) gives a CRC that does not
    depend on the message: the code's fixed residue."""
    rng = random.Random(6)
    seen = set()
    for _ in range(100):
        m = _rand_bytes(rng, rng.randrange(0, 200))
        c = orc.crc32c(m)
        seen.add(orc.crc32c(m + c.to_bytes(4, "little")))
    assert len(seen) == 1


def test_detects_every_single_bit_error(orc):
    rng = random.Random(7)
    m = bytearray(_rand_bytes(rng, 64))
    base = orc.crc32c(bytes(m))
    for bit in range(len(m) * 8):
        m[bit // 8] ^= 1 << (bit % 8)
        assert orc.crc32c(bytes(m)) != base
        m[bit // 8] ^= 1 << (bit % 8)


@pytest.mark.parametrize("burst", [2, 7, 17, 32])
def test_detects_bursts_up_to_32_bits(orc, burst):
    rng = random.Random(8 + burst)
    n = 48
    m = int.from_bytes(_rand_bytes(rng, n), "little")
    base = orc.crc32c(m.to_bytes(n, "little"))
    for _ in range(200):
        start = rng.randrange(0, n * 8 - burst + 1)
        pattern = (1 | (1 << (burst - 1))) | (rng.getrandbits(burst) if burst > 2 else 0)
        pattern &= (1 << burst) - 1
        pattern |= 1 | (1 << (burst - 1))
        e = m ^ (pattern << start)
        assert orc.crc32c(e.to_bytes(n, "little")) != base
