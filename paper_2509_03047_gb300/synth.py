"""Seeded synthetic optimizer states and fault injection.

This module only generates inputs: it holds none of the restoration sweep's
arithmetic (no checksum, no sum of squares, no layout).  Both the CUDA path's
tests/benchmark and the CPU oracle's tests draw their inputs from here.

The workloads stand in for the per-rank state that FlashRecovery restores from
a data-parallel replica (arXiv 2509.03047, Sec. III-E); the paper's own
training runs (7B/70B/175B on Ascend NPUs, Sec. IV) are private, so shapes
follow public model architectures and values follow the usual initial
distributions of mixed-precision Adam state:

* every parameter tensor contributes four buffers, in this order:
  bf16 weight, fp32 master weight, fp32 Adam m, fp32 Adam v;
* master ~ N(0, 0.02) (sigma is the standard deviation), weight = bf16(master)
  by round-to-nearest-even, then master := float(weight) so that the master
  equals the weight exactly;
* m ~ N(0, 1e-3); v = (N(0, 1e-3))^2 in fp32.

Integer randomness (sizes, fault positions) comes from splitmix64 (Steele,
Lea, Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014),
so fault positions are identical on every machine.  Float values come from
torch generators seeded per (seed, tensor, kind).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List, Sequence, Tuple

import numpy as np
import torch

KiB = 1024
MiB = 1024 * 1024
MASK64 = (1 << 64) - 1

DT_BYTES, DT_BF16, DT_F32 = 0, 1, 2
TORCH_DT = {DT_BF16: torch.bfloat16, DT_F32: torch.float32, DT_BYTES: torch.uint8}
ELEM_BYTES = {DT_BF16: 2, DT_F32: 4, DT_BYTES: 1}


# ---------------------------------------------------------------- splitmix64

class SplitMix64:
    """splitmix64: state += golden gamma; output = mix(state)."""

    def __init__(self, seed: int):
        self.state = seed & MASK64

    def next(self) -> int:
        self.state = (self.state + 0x9E3779B97F4A7C15) & MASK64
        z = self.state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
        return z ^ (z >> 31)

    def uniform(self) -> float:
        """A double in [0, 1) from the top 53 bits."""
        return (self.next() >> 11) * (1.0 / (1 << 53))

    def below(self, n: int) -> int:
        """Uniform integer in [0, n) by rejection (no modulo bias)."""
        if n <= 0:
            raise ValueError("n must be positive")
        limit = (1 << 64) - ((1 << 64) % n)
        while True:
            x = self.next()
            if x < limit:
                return x % n


def derive_seed(*parts: int) -> int:
    """A 64-bit seed for a sub-stream, mixed from integer parts."""
    h = 0x5EED
    for p in parts:
        h = SplitMix64(h ^ (p & MASK64)).next()
    return h


def distinct_positions(n: int, count: int, seed: int) -> np.ndarray:
    """`count` distinct integers uniform in [0, n), sorted ascending."""
    if count > n:
        raise ValueError("more positions than slots")
    rng = SplitMix64(seed)
    seen = set()
    while len(seen) < count:
        seen.add(rng.below(n))
    return np.array(sorted(seen), dtype=np.int64)


# ---------------------------------------------------------------- shapes

def tiny_shapes() -> List[Tuple[str, Tuple[int, ...]]]:
    """8 tensors, hidden 256, ffn 1024, vocab 2048, 2 layers: 1,050,880 params.

    Two full GPT blocks plus the embedding would be 2.1M parameters, more than
    the ~1.1M the workload asks for, so each layer keeps its fused QKV, the
    attention output projection and an MLP bias (1024), and a final norm."""
    shapes = [("tok_emb", (2048, 256))]
    for layer in range(2):
        shapes += [
            ("l%d.attn_qkv" % layer, (768, 256)),
            ("l%d.attn_out" % layer, (256, 256)),
            ("l%d.mlp_fc_bias" % layer, (1024,)),
        ]
    shapes.append(("ln_f", (256,)))
    return shapes


def gpt2_small_shapes() -> List[Tuple[str, Tuple[int, ...]]]:
    """GPT-2 small, 148 tensors, 124,439,808 params."""
    h, ffn, vocab, ctx, layers = 768, 3072, 50257, 1024, 12
    shapes = [("wte", (vocab, h)), ("wpe", (ctx, h))]
    for i in range(layers):
        p = "h%d." % i
        shapes += [
            (p + "ln_1.weight", (h,)), (p + "ln_1.bias", (h,)),
            (p + "attn.c_attn.weight", (h, 3 * h)), (p + "attn.c_attn.bias", (3 * h,)),
            (p + "attn.c_proj.weight", (h, h)), (p + "attn.c_proj.bias", (h,)),
            (p + "ln_2.weight", (h,)), (p + "ln_2.bias", (h,)),
            (p + "mlp.c_fc.weight", (h, ffn)), (p + "mlp.c_fc.bias", (ffn,)),
            (p + "mlp.c_proj.weight", (ffn, h)), (p + "mlp.c_proj.bias", (h,)),
        ]
    shapes += [("ln_f.weight", (h,)), ("ln_f.bias", (h,))]
    return shapes


def llama_shard_shapes(hidden: int, ffn: int, layers: int, vocab: int, n_kv: int,
                       head_dim: int, tp: int, with_head: bool) -> List[Tuple[str, Tuple[int, ...]]]:
    """One tensor-parallel rank of a Llama-3 model.

    q/o/gate/up/down and the embedding are split by `tp`; k and v keep
    n_kv*head_dim/tp rows (one KV head at tp=8); norms are replicated."""
    kv = n_kv * head_dim // tp
    shapes = [("embed", (vocab // tp, hidden))]
    for i in range(layers):
        p = "layers.%d." % i
        shapes += [
            (p + "attn_norm", (hidden,)),
            (p + "q_proj", (hidden // tp, hidden)),
            (p + "k_proj", (kv, hidden)),
            (p + "v_proj", (kv, hidden)),
            (p + "o_proj", (hidden, hidden // tp)),
            (p + "ffn_norm", (hidden,)),
            (p + "gate_proj", (ffn // tp, hidden)),
            (p + "up_proj", (ffn // tp, hidden)),
            (p + "down_proj", (hidden, ffn // tp)),
        ]
    if with_head:
        shapes += [("norm", (hidden,)), ("lm_head", (vocab // tp, hidden))]
    return shapes


def frag_sizes(count: int, lo: int, hi: int, seed: int) -> List[int]:
    """`count` byte sizes log-uniform in [lo, hi], rounded down to 4 bytes."""
    rng = SplitMix64(derive_seed(seed, 0xF7A6))
    a, b = math.log(lo), math.log(hi)
    out = []
    for _ in range(count):
        s = int(math.exp(a + rng.uniform() * (b - a)))
        out.append(max(4, s // 4 * 4))
    return out


# ---------------------------------------------------------------- configs

@dataclass
class Config:
    name: str
    chunk_bytes: int
    kind: str                      # "adam" (4 buffers per param tensor) or "frag"
    shapes: List[Tuple[str, Tuple[int, ...]]] = field(default_factory=list)
    frag: Tuple[int, int, int] = (0, 0, 0)  # (count, lo bytes, hi bytes)
    nan_count: int = 0             # NaNs injected into the state
    nonfinite_frac: float = 0.0    # frag: fraction of elements set to +-Inf/NaN
    flips: int = 0                 # bit flips injected into the packed buffer
    diff_chunks: int = 0           # chunks modified in the diff copy
    seed: int = 0

    def buffer_specs(self) -> List[Tuple[str, int, int]]:
        """(name, dtype, nbytes) of every buffer, in plan order."""
        specs = []
        if self.kind == "adam":
            for name, shape in self.shapes:
                n = int(np.prod(shape))
                specs += [(name + ".weight", DT_BF16, 2 * n), (name + ".master", DT_F32, 4 * n),
                          (name + ".adam_m", DT_F32, 4 * n), (name + ".adam_v", DT_F32, 4 * n)]
        else:
            cnt, lo, hi = self.frag
            for i, s in enumerate(frag_sizes(cnt, lo, hi, self.seed)):
                specs.append(("frag.%d" % i, DT_F32, s))
        return specs

    def params(self) -> int:
        return sum(int(np.prod(s)) for _, s in self.shapes)

    def state_bytes(self) -> int:
        return sum(b for _, _, b in self.buffer_specs())


def get_config(name: str) -> Config:
    if name == "tiny":
        return Config("tiny", 64 * KiB, "adam", tiny_shapes(), nan_count=3, flips=2)
    if name == "gpt2s":
        return Config("gpt2s", 1 * MiB, "adam", gpt2_small_shapes())
    if name == "l8b_tp8":
        return Config("l8b_tp8", 4 * MiB, "adam",
                      llama_shard_shapes(4096, 14336, 32, 128256, 8, 128, 8, True), flips=10)
    if name == "zero_frag":
        return Config("zero_frag", 256 * KiB, "frag", frag=(50000, 1 * KiB, 4 * MiB),
                      nonfinite_frac=1e-7, diff_chunks=100)
    if name == "zero_frag4g":
        return Config("zero_frag4g", 256 * KiB, "frag", frag=(50000, 1 * KiB, 512 * KiB),
                      nonfinite_frac=1e-7, diff_chunks=100)
    if name == "l70b_tp8pp4":
        return Config("l70b_tp8pp4", 16 * MiB, "adam",
                      llama_shard_shapes(8192, 28672, 20, 128256, 8, 128, 8, False),
                      flips=1000, nan_count=50)
    raise KeyError(name)


CONFIG_NAMES = ["tiny", "gpt2s", "l8b_tp8", "zero_frag", "l70b_tp8pp4"]


# ---------------------------------------------------------------- values

def _gen(device, *parts) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(derive_seed(*parts) & ((1 << 63) - 1))
    return g


def make_state(cfg: Config, device="cpu") -> List[torch.Tensor]:
    """The clean (fault-free) state buffers of `cfg`, flat 1-D tensors."""
    out: List[torch.Tensor] = []
    if cfg.kind == "adam":
        for t, (name, shape) in enumerate(cfg.shapes):
            n = int(np.prod(shape))
            master = torch.randn(n, generator=_gen(device, cfg.seed, t, 1), device=device,
                                 dtype=torch.float32) * 0.02
            weight = master.to(torch.bfloat16)
            master = weight.to(torch.float32)
            m = torch.randn(n, generator=_gen(device, cfg.seed, t, 2), device=device,
                            dtype=torch.float32) * 1e-3
            v = torch.randn(n, generator=_gen(device, cfg.seed, t, 3), device=device,
                            dtype=torch.float32) * 1e-3
            v = v * v
            out += [weight, master, m, v]
    else:
        for i, (name, dt, nbytes) in enumerate(cfg.buffer_specs()):
            out.append(torch.randn(nbytes // 4, generator=_gen(device, cfg.seed, i, 9), device=device,
                                   dtype=torch.float32))
    return out


def element_counts(tensors: Sequence[torch.Tensor]) -> List[int]:
    return [t.numel() for t in tensors]


def _locate(counts: Sequence[int], positions: np.ndarray):
    """Map global element positions to (buffer index, element index)."""
    starts = np.concatenate([[0], np.cumsum(np.asarray(counts, dtype=np.int64))])
    buf = np.searchsorted(starts, positions, side="right") - 1
    return buf, positions - starts[buf]


def nan_positions(cfg: Config, tensors: Sequence[torch.Tensor]) -> np.ndarray:
    total = sum(element_counts(tensors))
    if cfg.kind == "frag":
        count = int(round(cfg.nonfinite_frac * total))
    else:
        count = cfg.nan_count
    return distinct_positions(total, count, derive_seed(cfg.seed, 0xAA))


def inject_nonfinite(cfg: Config, tensors: List[torch.Tensor]) -> np.ndarray:
    """Write NaN (adam configs) or seeded +-Inf/NaN (frag) at seeded element
    positions, in place.  Returns the global positions."""
    pos = nan_positions(cfg, tensors)
    if pos.size == 0:
        return pos
    buf, idx = _locate(element_counts(tensors), pos)
    rng = SplitMix64(derive_seed(cfg.seed, 0xAB))
    for b, i in zip(buf.tolist(), idx.tolist()):
        t = tensors[b]
        if cfg.kind == "frag":
            val = [float("inf"), float("-inf"), float("nan")][rng.below(3)]
        else:
            val = float("nan")
        t[i] = val
    return pos


def flip_positions(packed_bytes: int, count: int, seed: int) -> np.ndarray:
    """`count` distinct bit positions uniform over all bits of the packed buffer."""
    if count == 0 or packed_bytes == 0:
        return np.zeros(0, dtype=np.int64)
    return distinct_positions(packed_bytes * 8, count, derive_seed(seed, 0xF1))


def apply_flips(buf: torch.Tensor, bit_positions: np.ndarray) -> None:
    """XOR single bits of a uint8 buffer (device or host), in place."""
    if bit_positions.size == 0:
        return
    byte = torch.as_tensor(bit_positions // 8, dtype=torch.int64, device=buf.device)
    mask = torch.as_tensor(1 << (bit_positions % 8), dtype=torch.uint8, device=buf.device)
    # positions are distinct bits, but two may share a byte: accumulate by XOR
    uniq, inv = torch.unique(byte, return_inverse=True)
    acc = torch.zeros(uniq.numel(), dtype=torch.uint8, device=buf.device)
    for j in range(mask.numel()):  # few flips: a plain loop is clear and fast enough
        acc[inv[j]] ^= mask[j]
    buf[uniq] ^= acc


def modify_for_diff(cfg: Config, tensors: List[torch.Tensor], chunks) -> np.ndarray:
    """Change one seeded element in each of `cfg.diff_chunks` seeded chunks of
    a copy of the state (in place on `tensors`).  `chunks` is a sequence of
    (tensor_idx, tensor_off, len, dtype) rows.  Returns the chunk ids."""
    ids = distinct_positions(len(chunks), cfg.diff_chunks, derive_seed(cfg.seed, 0xD1))
    rng = SplitMix64(derive_seed(cfg.seed, 0xD2))
    for c in ids.tolist():
        t_idx, off, length, dt = [int(x) for x in chunks[c]]
        esz = ELEM_BYTES[dt]
        e = off // esz + rng.below(length // esz)
        t = tensors[t_idx]
        if dt == DT_F32:
            bits = t.view(torch.int32)
            v = int(bits[e].item())
            if (v & 0x7F800000) == 0x7F800000:
                t[e] = 1.0
            else:
                bits[e] = v ^ 1  # a different finite value: lowest mantissa bit
        elif dt == DT_BF16:
            bits = t.view(torch.int16)
            v = int(bits[e].item()) & 0xFFFF
            if (v & 0x7F80) == 0x7F80:
                t[e] = 1.0
            else:
                nv = v ^ 1
                bits[e] = nv - 0x10000 if nv >= 0x8000 else nv
        else:
            bits = t.view(torch.uint8)
            bits[e] = int(bits[e].item()) ^ 1
    return ids
