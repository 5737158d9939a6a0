"""fr_fingerprint_static, the fingerprint entry point that allocates nothing.

It exists for callers that cannot allocate device memory -- typically a
recovery agent running inside a training process whose framework allocator
has reserved the whole GPU for the model and optimizer state.  Its plan tables
and scratch live in a fixed array inside the library, shared by every call.
This file runs last (pytest collects it after the others) so that a failure
here never hides the rest of the suite, and it passes both alone in a fresh
process and after every other test."""
import numpy as np
import pytest
import torch

from paper_2509_03047_gb300 import synth

import oracle
from gpu_helpers import Guarded, assert_tables_match, host_bytes, odd_tensors, table_np

pytestmark = pytest.mark.gpu

fr = pytest.importorskip("paper_2509_03047_gb300.flashrec")


def _static_table(tensors, chunk):
    n = fr.Plan(tensors, chunk).n_chunks
    out = Guarded(n * 16)
    fr.fr_fingerprint_static(tensors, chunk, out.buf)
    torch.cuda.synchronize()
    out.check("static fingerprint table")
    return out.buf


def test_static_entry_point_matches_plan_on_three_calls_in_a_row():
    # call 1: the tiny workload, with its injected NaNs
    cfg = synth.get_config("tiny")
    a = synth.make_state(cfg, "cuda")
    synth.inject_nonfinite(cfg, a)
    # call 2: a different list -- misaligned views, mixed types, ragged tails
    base = torch.randn((3 << 20) + 64, device="cuda")
    b = [base[1:1 + 700000], base[800001:800001 + 333333].to(torch.bfloat16).contiguous(),
         base[2000000:2000000 + 1000003], torch.randint(0, 256, (99999,), device="cuda", dtype=torch.uint8)]
    # call 3: every (element type, alignment) class, awkward sizes
    c = odd_tensors(4, 2)
    for tensors, chunk in [(a, cfg.chunk_bytes), (b, 12288), (c, 4096)]:
        want = fr.Plan(tensors, chunk).fingerprint()
        got = _static_table(tensors, chunk)
        assert got.numel() == want.numel()
        assert_tables_match(table_np(got), table_np(want), "static vs plan")
        # and directly against the oracle, every entry
        dtypes = [fr.fr_dtype_of(t) for t in tensors]
        assert_tables_match(table_np(got), oracle.fingerprint(host_bytes(tensors), dtypes, chunk), "static vs oracle")


def test_static_entry_point_rejects_inputs_beyond_its_limit():
    t = torch.zeros(4 * (fr.FR_STATIC_MAX_CHUNKS + 1), dtype=torch.uint8, device="cuda")
    out = torch.empty(16 * (fr.FR_STATIC_MAX_CHUNKS + 1), dtype=torch.uint8, device="cuda")
    with pytest.raises(fr.FlashrecError) as e:
        fr.fr_fingerprint_static([t], 4, out)
    assert e.value.status == fr.FR_ERR_INVALID_ARG
    assert "FR_STATIC_MAX_CHUNKS" in fr.fr_last_error()
    # the largest allowed input still works
    ok = t[: 4 * fr.FR_STATIC_MAX_CHUNKS]
    got = _static_table([ok], 4)
    want = fr.Plan([ok], 4).fingerprint()
    assert torch.equal(got, want)


def test_static_entry_point_refuses_a_stream_under_capture():
    # a graph replay would upload whatever tables the latest call left in the
    # library's host buffer, so the call refuses capture and enqueues nothing
    t = torch.randn(8192, device="cuda")
    out = torch.empty(16 * 2, dtype=torch.uint8, device="cuda")
    want = fr.Plan([t], 16384).fingerprint()
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        with pytest.raises(fr.FlashrecError) as e:
            fr.fr_fingerprint_static([t], 16384, out, stream=s)
    assert e.value.status == fr.FR_ERR_INVALID_ARG
    assert "captured" in fr.fr_last_error()
    # the same call outside the capture works
    assert torch.equal(_static_table([t], 16384), want)
