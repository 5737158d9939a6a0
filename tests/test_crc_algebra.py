"""The GF(2) identities the kernels compute CRC-32C with, restated in plain
Python and checked against the oracle's bytewise CRC-32C.  No GPU.

The kernels never run the textbook byte-at-a-time CRC.  The sweep treats the
128 words of a 512-byte block as 128 interleaved streams and folds them, lane
by lane and then over a shuffle tree, at the end of a piece; finalize joins
pieces by shifts, reads a tail as the end of a zero-led 512-byte window whose
words are strided over the 32 lanes, and computes the 60-byte header CRC
from one word per lane.  Each test below is the arithmetic of one of those
steps (same exponents, lane mapping and fold order as the CUDA code, in the
reflected representation of gf2.cuh: bit 31 of a word is x^0), so a wrong
exponent, lane or order fails it.
"""
import numpy as np
import pytest

import oracle

P = 0x82F63B78  # x^32 mod P(x), reflected
ONE = 0x80000000  # the polynomial 1


def mul_x(r):
    return (r >> 1) ^ (P if r & 1 else 0)


def mulmod(a, b):
    r = 0
    for k in range(32):
        if a & (ONE >> k):
            r ^= b
        b = mul_x(b)
    return r


def xpow(n):
    r, base = ONE, mul_x(ONE)
    while n:
        if n & 1:
            r = mulmod(r, base)
        base = mulmod(base, base)
        n >>= 1
    return r


def div_x(r):
    return (((r ^ P) << 1) | 1) & 0xFFFFFFFF if r & ONE else (r << 1) & 0xFFFFFFFF


def xpow_neg(n):
    r, base = ONE, div_x(ONE)
    while n:
        if n & 1:
            r = mulmod(r, base)
        base = mulmod(base, base)
        n >>= 1
    return r


def crc_of_raw(raw, n):
    """CRC-32C of an n-byte message from its raw CRC (preset 0, no final XOR)."""
    return raw ^ mulmod(0xFFFFFFFF, xpow(8 * n)) ^ 0xFFFFFFFF


def words(b):
    return [int(w) for w in np.frombuffer(bytes(b), dtype="<u4")]


def rand_bytes(rng, n):
    return rng.integers(0, 256, n, dtype=np.uint8).tobytes()


def want_crc(data):
    return oracle.crc32c(np.frombuffer(data, dtype=np.uint8)) if data else 0


def test_helpers_against_the_check_value():
    assert crc_of_raw(0, 0) == 0  # the empty message
    # the byte-serial register run: each byte enters as b * x^8 ... via xor and 8 shifts
    r = 0
    for c in b"123456789":
        r ^= c
        for _ in range(8):
            r = mul_x(r)
    assert crc_of_raw(r, 9) == 0xE3069283 == want_crc(b"123456789")
    assert mulmod(xpow(100), xpow_neg(100)) == ONE


@pytest.mark.parametrize("n_blocks", [1, 2, 5])
def test_braided_streams_folded_lane_by_lane_then_over_a_shuffle_tree(n_blocks):
    # sweep: lane l owns streams 4l..4l+3; a stream steps s <- (s ^ w) * x^4096;
    # at the piece end each lane folds its four streams by x^32 (Horner), a
    # five-level tree joins lane l + d into lane l with x^(128 d), and x^(-32*127)
    # removes the braid's offset
    rng = np.random.default_rng(n_blocks)
    data = rand_bytes(rng, 512 * n_blocks)
    x4096, x32 = xpow(4096), xpow(32)
    s = [0] * 128
    for b in range(n_blocks):
        w = words(data[512 * b: 512 * (b + 1)])
        for j in range(128):
            s[j] = mulmod(s[j] ^ w[j], x4096)
    v = []
    for lane in range(32):
        acc = 0
        for q in range(4):
            acc = mulmod(acc, x32) ^ s[4 * lane + q]
        v.append(acc)
    d = 1
    while d < 32:
        v = [mulmod(v[lane], xpow(128 * d)) ^ (v[lane + d] if lane + d < 32 else 0) for lane in range(32)]
        d *= 2
    raw = mulmod(v[0], xpow_neg(32 * 127))
    assert crc_of_raw(raw, len(data)) == want_crc(data)


def test_pieces_joined_by_shifts():
    # finalize: raw(A || B) = raw(A) * x^(8|B|) ^ raw(B); a piece followed by n
    # more bytes of its chunk's body takes the multiplier x^(8n)
    rng = np.random.default_rng(1)
    pieces = [rand_bytes(rng, 512 * k) for k in (3, 1, 2)]

    def raw(b):
        r = 0
        for c in b:
            r ^= c
            for _ in range(8):
                r = mul_x(r)
        return r

    total = 0
    after = sum(len(p) for p in pieces)
    for p in pieces:
        after -= len(p)
        total ^= mulmod(raw(p), xpow(8 * after))
    data = b"".join(pieces)
    assert crc_of_raw(total, len(data)) == want_crc(data)


def lane_table():
    """(n << 4k) * x^(32 (32 - l)) for nibble position k, value n, lane l."""
    return {(k, n, lane): mulmod(n << (4 * k), xpow(32 * (32 - lane)))
            for lane in range(32) for k in range(8) for n in range(16)}


@pytest.fixture(scope="module")
def lm():
    return lane_table()


def lane_mul(lm, a, lane):
    r = 0
    for k in range(8):
        r ^= lm[(k, (a >> (4 * k)) & 15, lane)]
    return r


def test_lane_table_multiplies_by_the_lane_shift(lm):
    rng = np.random.default_rng(2)
    for lane in range(32):
        a = int(rng.integers(0, 1 << 32))
        assert lane_mul(lm, a, lane) == mulmod(a, xpow(32 * (32 - lane)))


@pytest.mark.parametrize("body_blocks", [0, 1, 2])
@pytest.mark.parametrize("tail", [1, 2, 3, 4, 6, 64, 100, 128, 130, 252, 256, 384, 500, 508, 510, 511])
def test_tail_as_a_word_strided_window(lm, body_blocks, tail):
    # finalize: the tail is the end of a 512-byte window led by 512 - tail
    # zero bytes; window word i is word i // 32 of lane i % 32; when the tail
    # is a whole number of words the body's raw CRC is XORed into its first
    # word, else the body is shifted by x^(8 tail); lane l combines its words as
    # sum_q w_q x^(1024 (3 - q)) (x^1024 twice, x^2048 once), takes its shift
    # x^(32 (32 - l)), and the lanes are XORed
    rng = np.random.default_rng(1000 * body_blocks + tail)
    body = rand_bytes(rng, 512 * body_blocks)
    t = rand_bytes(rng, tail)
    data = body + t
    z = 512 - tail
    win = words(bytes(z) + t)
    # the body's raw CRC, from the oracle's CRC of the body (preset and final
    # XOR undone: the term is its own inverse)
    raw_body = crc_of_raw(want_crc(body), len(body)) if body else 0
    fold = tail % 4 == 0
    if fold and body:
        win[z // 4] ^= raw_body
    x1024, x2048 = xpow(1024), xpow(2048)
    joined = 0
    for lane in range(32):
        w = [win[32 * q + lane] for q in range(4)]
        h = mulmod(mulmod(w[0], x1024) ^ w[1], x2048) ^ (mulmod(w[2], x1024) ^ w[3])
        joined ^= lane_mul(lm, h, lane)
    raw = joined if (fold or not body) else (mulmod(raw_body, xpow(8 * tail)) ^ joined)
    assert crc_of_raw(raw, len(data)) == want_crc(data)


def test_header_crc_from_one_word_per_lane(lm):
    # finalize: header word k (of 15) sits in lane 17 + k, whose shift
    # x^(32 (15 - k)) is exactly the word's; the lanes are XORed
    rng = np.random.default_rng(3)
    for _ in range(5):
        h = [int(x) for x in rng.integers(0, 1 << 32, 15, dtype=np.uint64)]
        raw = 0
        for k in range(15):
            raw ^= lane_mul(lm, h[k], 17 + k)
        data = np.array(h, dtype="<u4").tobytes()
        assert crc_of_raw(raw, 60) == want_crc(data)
