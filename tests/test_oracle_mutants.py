"""The pins pin: copies of the oracle with one planted mistake each (a wrong
constant, shift, bound, field, mask or skipped check) are compiled on the CPU,
and for every one of them at least one pin test must fail.  The planted
mistakes live only in temporary copies; the real oracle is untouched."""
import os
import subprocess
import tempfile

import pytest

import oracle
import test_oracle_crc as tcrc
import test_oracle_fp as tfp
import test_oracle_pack as tpack

SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

MUTANTS = {
    "polynomial": ("#define OR_CRC32C_POLY 0x82F63B78u", "#define OR_CRC32C_POLY 0x82F63B79u"),
    "table_shift": ("r = table[(r ^ p[i]) & 0xFFu] ^ (r >> 8);", "r = table[(r ^ p[i]) & 0xFFu] ^ (r >> 7);"),
    "combine_len": ("for (uint64_t i = 0; i < len_b; ++i) r = table[r & 0xFFu] ^ (r >> 8);",
                    "for (uint64_t i = 1; i < len_b; ++i) r = table[r & 0xFFu] ^ (r >> 8);"),
    "square_in_fp32": ("s = s + x * x; /* the product", "s = s + (double)((float)x * (float)x); /* the product"),
    "exponent_mask": ("if ((bits & 0x7F800000u) == 0x7F800000u) {", "if ((bits & 0x7F000000u) == 0x7F000000u) {"),
    "bf16_shift": ("double x = (double)float_from_bits((uint32_t)bits << 16);",
                   "double x = (double)float_from_bits((uint32_t)bits << 15);"),
    "bf16_nan_summed": ("if ((bits & 0x7F80u) == 0x7F80u) {\n        bad += 1;\n      } else {",
                        "if ((bits & 0x7F80u) == 0x7F80u) {\n        bad += 1;\n      } {"),
    "header_field": ("store_le64(h + 24, ch->tensor_off);", "store_le64(h + 24, ch->len);"),
    "header_crc_span": ("store_le32(h + 60, or_crc32c(h, 60));", "store_le32(h + 60, or_crc32c(h, 56));"),
    "payload_align": ("off += align_up(len, OR_PAYLOAD_ALIGN);", "off += align_up(len, 128);"),
    "tail_length": ("if (len > chunk_bytes) len = chunk_bytes;", "if (len >= chunk_bytes) len = chunk_bytes - 4;"),
    "no_padding_check": ("for (uint64_t i = ch->len; i < pad_end; ++i)\n    if (payload[i] != 0) bad = 1;",
                         "for (uint64_t i = ch->len; i < pad_end; ++i)\n    if (0) bad = 1;"),
    "no_gap_check": ("for (uint64_t i = 0; i < gap_len; ++i)\n    if (gap[i] != 0) bad = 1;",
                     "for (uint64_t i = 0; i < gap_len; ++i)\n    if (0) bad = 1;"),
    "no_offset_check": ("if (load_le64(h + 24) != ch->tensor_off) bad = 1;", ""),
    "no_chunk_id_check": ("if (load_le64(h + 8) != chunk_id) bad = 1;", ""),
    "copy_only_good": ("memcpy(tensors[ch->tensor_idx] + ch->tensor_off, payload, (size_t)ch->len);",
                       "if (!bad) memcpy(tensors[ch->tensor_idx] + ch->tensor_off, payload, (size_t)ch->len);"),
    "diff_crc_only": ("if (memcmp(&a[c], &b[c], sizeof(or_fp)) != 0) {", "if (memcmp(&a[c], &b[c], 4) != 0) {"),
}


def _pins():
    """Every CPU pin test, as (name, callable taking the oracle module)."""
    out = []
    for mod in (tcrc, tfp, tpack):
        for name in dir(mod):
            fn = getattr(mod, name)
            if not name.startswith("test_") or not callable(fn):
                continue
            params = getattr(fn, "pytestmark", [])
            argsets = [()]
            for m in params:
                if m.name == "parametrize":
                    argsets = [(v if isinstance(v, tuple) else (v,)) for v in m.args[1]]
            for args in argsets:
                out.append(("%s.%s%s" % (mod.__name__, name, args), fn, args))
    return out


@pytest.fixture(scope="module")
def tmpdir_mut():
    with tempfile.TemporaryDirectory() as d:
        yield d


@pytest.mark.parametrize("mutant", sorted(MUTANTS))
def test_every_planted_mistake_fails_a_pin(mutant, tmpdir_mut):
    old, new = MUTANTS[mutant]
    src = open(SRC).read()
    assert src.count(old) == 1, "mutant anchor must be unique: %s" % mutant
    path_c = os.path.join(tmpdir_mut, mutant + ".c")
    with open(path_c, "w") as f:
        f.write(src.replace(old, new))
    so = os.path.join(tmpdir_mut, mutant + ".so")
    subprocess.check_call(["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fPIC", "-shared", "-w",
                           "-I", os.path.dirname(SRC), path_c, "-o", so])
    oracle.use_library(so)
    caught = []
    try:
        for name, fn, args in _pins():
            try:
                import inspect

                if "orc" in inspect.signature(fn).parameters:
                    fn(oracle, *args)
                else:
                    fn(*args)
            except Exception:  # an assertion or any other failure counts
                caught.append(name)
                break
    finally:
        oracle.use_library(None)
    assert caught, "no pin caught the planted mistake %r" % mutant
