"""The seeded workload generator: sizes follow from the model shapes, the
generator is deterministic, and fault positions are distinct and in range."""
import numpy as np
import torch

from paper_2509_03047_gb300 import synth


def test_parameter_counts_from_shapes():
    # closed forms of the architectures' tensor shapes
    assert synth.get_config("tiny").params() == 1_050_880
    assert synth.get_config("gpt2s").params() == 124_439_808
    assert synth.get_config("l8b_tp8").params() == 1_004_015_616
    assert synth.get_config("l70b_tp8pp4").params() == 2_270_756_864
    assert len(synth.get_config("gpt2s").shapes) == 148
    assert len(synth.get_config("l8b_tp8").shapes) == 291
    assert len(synth.get_config("l70b_tp8pp4").shapes) == 181


def test_state_bytes_are_14_per_param():
    for name in ["tiny", "gpt2s", "l8b_tp8", "l70b_tp8pp4"]:
        cfg = synth.get_config(name)
        assert cfg.state_bytes() == 14 * cfg.params()
    assert synth.get_config("tiny").state_bytes() == 14_712_320


def test_frag_sizes():
    cfg = synth.get_config("zero_frag")
    specs = cfg.buffer_specs()
    sizes = np.array([b for _, _, b in specs])
    assert len(specs) == 50_000
    assert sizes.min() >= 1024 - 4 and sizes.max() <= 4 * 1024 * 1024
    assert (sizes % 4 == 0).all()
    # log-uniform: the median is near the geometric mean sqrt(1 KiB * 4 MiB) = 64 KiB
    assert 50_000 < np.median(sizes) < 82_000
    assert synth.frag_sizes(10, 1024, 4 << 20, 0) == synth.frag_sizes(10, 1024, 4 << 20, 0)


def test_splitmix_determinism_and_range():
    a = synth.distinct_positions(1000, 50, 7)
    b = synth.distinct_positions(1000, 50, 7)
    assert np.array_equal(a, b)
    assert len(set(a.tolist())) == 50 and a.min() >= 0 and a.max() < 1000
    assert np.all(np.diff(a) > 0)
    r = synth.SplitMix64(3)
    xs = [r.below(7) for _ in range(2000)]
    assert set(xs) == set(range(7))


def test_tiny_state_distributions():
    cfg = synth.get_config("tiny")
    st = synth.make_state(cfg, "cpu")
    assert len(st) == 32
    w, m, am, av = st[0], st[1], st[2], st[3]
    assert w.dtype == torch.bfloat16 and m.dtype == torch.float32
    assert torch.equal(w.float(), m)
    assert abs(m.std().item() - 0.02) < 0.001
    assert abs(am.std().item() - 1e-3) < 1e-4
    assert (av >= 0).all()
    st2 = synth.make_state(cfg, "cpu")
    assert all(torch.equal(x.view(torch.uint8), y.view(torch.uint8)) for x, y in zip(st, st2))


def test_nan_injection_count():
    cfg = synth.get_config("tiny")
    st = synth.make_state(cfg, "cpu")
    pos = synth.inject_nonfinite(cfg, st)
    assert pos.size == 3
    n_nan = sum(int(torch.isnan(t.float()).sum()) for t in st)
    assert n_nan == 3


def test_apply_flips_xors_bits():
    buf = torch.zeros(16, dtype=torch.uint8)
    synth.apply_flips(buf, np.array([0, 1, 9, 127]))
    assert buf.tolist()[:2] == [3, 2] and buf[15].item() == 128
    synth.apply_flips(buf, np.array([0, 1, 9, 127]))
    assert int(buf.sum()) == 0
