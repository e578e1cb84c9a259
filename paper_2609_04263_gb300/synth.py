"""Seeded synthetic inputs for the packed-cache attention step.

This module holds random-number recipes only: no quantizer, projection,
rotation or attention arithmetic lives here, so both the CUDA path and the CPU
oracle can be fed from it without sharing any of the method's code.

Workload shapes follow the attention layers of the models the paper evaluates
(TinyLlama-1.1B, Llama-3.1-8B and a 12B-class Gemma-like shape, Section 4), with
the cache formats of Section 3.1.  Hidden states stand in for the WikiText
activations the paper calibrates and evaluates on (not available here):
N(0, 1) with 1% of channels scaled x20 as fixed outlier channels, or a
heavy-tailed Student-t (nu = 4).  Base weights are N(0, 0.02), LoRA A is
N(0, 0.02) and LoRA B is N(0, 0.01).
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

FMT_FLOAT, FMT_AFFINE, FMT_SYMMETRIC, FMT_KIVI, FMT_KVARN = range(5)
FMT_NAMES = {FMT_FLOAT: "float", FMT_AFFINE: "affine", FMT_SYMMETRIC: "symmetric",
             FMT_KIVI: "kivi", FMT_KVARN: "kvarn"}


@dataclasses.dataclass(frozen=True)
class Workload:
    """One benchmarked attention-stack shape and its cache format."""
    name: str
    dtype: str              # activation / weight dtype: "f32" or "bf16"
    layers: int
    d_in: int               # hidden size
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    rope_base: float
    batch: int
    prefill: int            # prompt tokens per sequence
    decode: int             # decode steps after the prompt
    fmt: int
    key_bits: int
    value_bits: int
    group_size: int
    residual_tokens: int = 0   # KIVI full-precision window
    sink_tokens: int = 0       # KVarN protected prefix
    norm_iters: int = 0        # KVarN dual-axis normalisation iterations
    rank: int = 8              # LoRA rank on each of Q, K, V
    alpha_over_r: float = 2.0
    hidden: str = "normal"     # "normal" or "student_t4"
    outlier_frac: float = 0.0

    @property
    def max_tokens(self) -> int:
        return self.prefill + self.decode

    @property
    def n_out(self) -> int:
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim


# The five workloads.  Sizes are the ones the method is evaluated at; the
# 12B-class shape uses RoPE base 10000 because no base is stated for it.
WORKLOADS = {
    "single_layer_f32": Workload(
        name="single_layer_f32", dtype="f32", layers=1, d_in=256, n_q_heads=4,
        n_kv_heads=4, head_dim=64, rope_base=10000.0, batch=1, prefill=512,
        decode=64, fmt=FMT_AFFINE, key_bits=4, value_bits=4, group_size=32,
        rank=8),
    "tinyllama_affine4": Workload(
        name="tinyllama_affine4", dtype="bf16", layers=22, d_in=2048,
        n_q_heads=32, n_kv_heads=4, head_dim=64, rope_base=10000.0, batch=4,
        prefill=2048, decode=256, fmt=FMT_AFFINE, key_bits=4, value_bits=4,
        group_size=32, rank=16, outlier_frac=0.01),
    "tinyllama_sym2": Workload(
        name="tinyllama_sym2", dtype="bf16", layers=22, d_in=2048,
        n_q_heads=32, n_kv_heads=4, head_dim=64, rope_base=10000.0, batch=8,
        prefill=4096, decode=1024, fmt=FMT_SYMMETRIC, key_bits=2, value_bits=2,
        group_size=32, rank=64, outlier_frac=0.01),
    "llama8b_kivi": Workload(
        name="llama8b_kivi", dtype="bf16", layers=32, d_in=4096, n_q_heads=32,
        n_kv_heads=8, head_dim=128, rope_base=500000.0, batch=16, prefill=8192,
        decode=64, fmt=FMT_KIVI, key_bits=2, value_bits=2, group_size=32,
        residual_tokens=128, rank=16, outlier_frac=0.01),
    "gemma12b_kvarn": Workload(
        name="gemma12b_kvarn", dtype="bf16", layers=48, d_in=3840, n_q_heads=16,
        n_kv_heads=8, head_dim=256, rope_base=10000.0, batch=4, prefill=8192,
        decode=512, fmt=FMT_KVARN, key_bits=4, value_bits=2, group_size=64,
        sink_tokens=128, norm_iters=8, rank=32, hidden="student_t4"),
}


def outlier_channels(d_in: int, frac: float, seed: int) -> np.ndarray:
    """Indices of the fixed outlier channels (seeded permutation)."""
    n = int(round(frac * d_in))
    if n == 0:
        return np.zeros(0, dtype=np.int64)
    rng = np.random.default_rng([seed, 7919])
    return np.sort(rng.permutation(d_in)[:n])


def hidden_states(shape, kind: str = "normal", outlier_frac: float = 0.0,
                  seed: int = 0, stream: int = 0) -> np.ndarray:
    """Hidden states [..., d_in] as float32.

    `stream` selects an independent draw (e.g. one per decode step) while the
    outlier channels stay fixed for a given seed.
    """
    rng = np.random.default_rng([seed, 1, stream])
    if kind == "normal":
        x = rng.standard_normal(shape, dtype=np.float64)
    elif kind == "student_t4":
        x = rng.standard_t(4.0, size=shape)
    else:
        raise ValueError(kind)
    idx = outlier_channels(shape[-1], outlier_frac, seed)
    if idx.size:
        x[..., idx] *= 20.0
    return x.astype(np.float32)


def layer_weights(wl: Workload, layer: int, seed: int = 0, rank=None):
    """Frozen W_qkv and LoRA (A, B) for one layer, float32.

    W_qkv is [(Hq + 2 Hkv) D, d_in] with the Q rows first, then K, then V.
    LoRA for projection p has A_p [r, d_in] and B_p [d_out_p, r].
    """
    r = wl.rank if rank is None else rank
    rng = np.random.default_rng([seed, 2, layer])
    D = wl.head_dim
    w = (0.02 * rng.standard_normal((wl.n_out, wl.d_in))).astype(np.float32)
    outs = {"q": wl.n_q_heads * D, "k": wl.n_kv_heads * D, "v": wl.n_kv_heads * D}
    lora = {}
    for p in "qkv":
        if r == 0:
            lora[p] = None
            continue
        a = (0.02 * rng.standard_normal((r, wl.d_in))).astype(np.float32)
        b = (0.01 * rng.standard_normal((outs[p], r))).astype(np.float32)
        lora[p] = (a, b)
    return w, lora


def nf4_base(wl: Workload, layer: int, seed: int = 0):
    """A frozen NF4 base for one layer: codes [(Hq + 2 Hkv) D, d_in / 2]
    (uint8, two 4-bit codes per byte, the even input in the low nibble) and
    absmax [(Hq + 2 Hkv) D, d_in / 64] (float32).

    NF4 levels are normal quantiles of equal probability, so the codes of
    normally distributed weights are uniform over the 16 levels: the codes
    are drawn uniformly; each block's absmax is the largest magnitude of 64
    draws of N(0, 0.02), the scale of the bf16 bases above.
    """
    rng = np.random.default_rng([seed, 6, layer])
    n, d_in = wl.n_out, wl.d_in
    codes = rng.integers(0, 256, size=(n, d_in // 2), dtype=np.uint8)
    absmax = np.abs(0.02 * rng.standard_normal((n, d_in // 64, 64))).max(axis=-1)
    return codes, absmax.astype(np.float32)


def kv_states(shape, seed: int = 0, stream: int = 0,
              channel_spread: float = 2.0) -> np.ndarray:
    """Key/value-like tensors [B, H, L, D] for exercising the cache alone.

    Each channel gets its own scale (log-uniform in [1/spread, spread]) and
    offset (N(0, 0.25)), which gives the per-channel structure real keys have
    at the unit scale of projected activations.
    """
    rng = np.random.default_rng([seed, 3, stream])
    D = shape[-1]
    crng = np.random.default_rng([seed, 4])
    scale = np.exp(crng.uniform(-math.log(channel_spread), math.log(channel_spread), D))
    offset = crng.normal(0.0, 0.25, D)
    x = rng.standard_normal(shape) * scale + offset
    return x.astype(np.float32)


def queries(shape, seed: int = 0, stream: int = 0) -> np.ndarray:
    rng = np.random.default_rng([seed, 5, stream])
    return rng.standard_normal(shape).astype(np.float32)
