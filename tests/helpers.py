"""Shared helpers of the parity tests: cache construction on both sides and
plane comparison restricted to live rows."""
from __future__ import annotations

import numpy as np
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import synth

ACT = {"bf16": torch.bfloat16, "f32": torch.float32}

# small formats used across the parity tests
FORMATS = {
    "float": dict(fmt=O.FMT_FLOAT, key_bits=4, value_bits=4, group_size=32),
    "affine4": dict(fmt=O.FMT_AFFINE, key_bits=4, value_bits=4, group_size=32),
    "affine2": dict(fmt=O.FMT_AFFINE, key_bits=2, value_bits=2, group_size=32),
    "affine8_g64": dict(fmt=O.FMT_AFFINE, key_bits=8, value_bits=8, group_size=64),
    "affine8": dict(fmt=O.FMT_AFFINE, key_bits=8, value_bits=8, group_size=32),
    "sym8": dict(fmt=O.FMT_SYMMETRIC, key_bits=8, value_bits=8, group_size=32),
    "affine4_g128": dict(fmt=O.FMT_AFFINE, key_bits=4, value_bits=2, group_size=128),
    "sym2": dict(fmt=O.FMT_SYMMETRIC, key_bits=2, value_bits=2, group_size=32),
    "sym4": dict(fmt=O.FMT_SYMMETRIC, key_bits=4, value_bits=4, group_size=32),
    "sym4_g8": dict(fmt=O.FMT_SYMMETRIC, key_bits=4, value_bits=8, group_size=8),
    "affine2_g16": dict(fmt=O.FMT_AFFINE, key_bits=2, value_bits=4, group_size=16),
    "kivi2": dict(fmt=O.FMT_KIVI, key_bits=2, value_bits=2, group_size=32,
                  residual_tokens=128),
    "kivi_r0": dict(fmt=O.FMT_KIVI, key_bits=2, value_bits=4, group_size=32,
                    residual_tokens=0),
    "kivi_g64": dict(fmt=O.FMT_KIVI, key_bits=4, value_bits=2, group_size=64,
                     residual_tokens=64),
    "kivi_k4": dict(fmt=O.FMT_KIVI, key_bits=4, value_bits=2, group_size=32,
                    residual_tokens=32),
    "kivi_k8": dict(fmt=O.FMT_KIVI, key_bits=8, value_bits=4, group_size=32,
                    residual_tokens=0),
    "kivi4": dict(fmt=O.FMT_KIVI, key_bits=4, value_bits=4, group_size=32,
                  residual_tokens=64),
    "kvarn": dict(fmt=O.FMT_KVARN, key_bits=4, value_bits=2, group_size=64,
                  sink_tokens=128, norm_iters=8),
    "kvarn_small": dict(fmt=O.FMT_KVARN, key_bits=4, value_bits=2, group_size=32,
                        sink_tokens=40, norm_iters=8),
}


def oracle_cache(spec, B, H, D, Tmax, act):
    kw = dict(spec)
    fmt = kw.pop("fmt")
    return O.OracleCache(fmt, batch=B, kv_heads=H, head_dim=D, max_tokens=Tmax, act=act, **kw)


def gpu_cache(spec, B, H, Hq, D, Tmax, act):
    from paper_2609_04263_gb300 import api
    kw = dict(spec)
    fmt = kw.pop("fmt")
    desc = api.make_desc(fmt, kw.get("key_bits", 4), kw.get("value_bits", 4),
                         kw.get("group_size", 32), B, H, Hq, D, Tmax, ACT[act],
                         residual_tokens=kw.get("residual_tokens", 0),
                         sink_tokens=kw.get("sink_tokens", 0),
                         norm_iters=kw.get("norm_iters", 8))
    return api.Cache(desc)


def kv_pair(B, H, L, D, act, seed=0, stream=0, device="cuda"):
    """Seeded k, v: torch tensors on the device and the same values as fp32
    numpy arrays for the oracle."""
    k = synth.kv_states((B, H, L, D), seed=seed, stream=2 * stream)
    v = synth.kv_states((B, H, L, D), seed=seed + 1000, stream=2 * stream + 1)
    kt = torch.from_numpy(k).to(ACT[act])
    vt = torch.from_numpy(v).to(ACT[act])
    return (kt.to(device), vt.to(device), kt.float().numpy(), vt.float().numpy())


def live(name, arr, oc):
    """Rows of a plane that hold live tokens (oc: the oracle cache state)."""
    T, G = oc.T, oc.G
    if name in ("k_row", "v_row"):
        arr = arr.reshape(arr.shape[0], arr.shape[1], -1)
    if oc.fmt == O.FMT_KIVI:
        tq = O.kivi_quantized_prefix(T, oc.R, G)
        if name.endswith("_full"):
            ring = oc.R + G
            return np.stack([arr[:, :, t % ring] for t in range(tq, T)], 2) if T > tq else arr[:, :, :0]
        if name in ("k_scale", "k_zero"):
            return arr[:, :, :tq // G]
        return arr[:, :, :tq]
    if oc.fmt == O.FMT_KVARN:
        nb = O.kvarn_blocks(T, oc.S, G)
        if name.endswith("_pend"):
            ts = range(oc.S + nb * G, T)
            return np.stack([arr[:, :, (t - oc.S) % G] for t in ts], 2) if len(ts) else arr[:, :, :0]
        if name.endswith("_col"):
            return arr[:, :, :nb]
        if name.endswith("_full"):
            return arr[:, :, :min(T, oc.S)]
        return arr[:, :, :nb * G]
    return arr[:, :, :T]


def to_numpy_plane(t: torch.Tensor) -> np.ndarray:
    if t.dtype == torch.bfloat16:
        return t.float().cpu().numpy()
    return t.cpu().numpy()


def compare_planes(gc, oc):
    """Bit-exact comparison of every oracle plane with the GPU plane."""
    gp = gc.planes()
    assert gp["_tokens"] == oc.T
    for name, ref in oc.planes.items():
        if ref.size == 0:
            continue
        assert name in gp, f"plane {name} missing on the GPU side"
        got = to_numpy_plane(gp[name])
        a, b = live(name, got, oc), live(name, ref, oc)
        assert a.shape == b.shape, (name, a.shape, b.shape)
        if a.dtype == np.float16:
            same = np.array_equal(a.view(np.uint16), b.view(np.uint16))
        elif a.dtype == np.float32:
            same = np.array_equal(a.view(np.uint32), b.astype(np.float32).view(np.uint32))
        else:
            same = np.array_equal(a, b)
        if not same:
            diff = np.argwhere(a.view(np.uint8) != b.view(np.uint8)) if a.dtype != np.float32 \
                else np.argwhere(a != b)
            raise AssertionError(f"plane {name}: {len(diff)} mismatches, first at {diff[:3].tolist()}")


def check_projection(got, ref, act, what=""):
    """Projection parity per (sequence, head): the max-abs difference from the
    oracle's fp64 result rounded to the activation dtype, over that head's
    largest oracle value, within 1e-2 (bf16) or 1e-5 (fp32).
    got (numpy, the GPU output as fp32) and ref (fp64): [B, H, L, D]."""
    tol = 1e-5 if act == "f32" else 1e-2
    r = O.round_to(ref, act).astype(np.float64)
    err = np.abs(np.asarray(got, dtype=np.float64) - r).max(axis=(2, 3))
    rel = err / np.maximum(np.abs(ref).max(axis=(2, 3)), 1e-30)
    worst = tuple(int(i) for i in np.unravel_index(int(rel.argmax()), rel.shape))
    assert rel.max() <= tol, f"{what}: (sequence, head) {worst} relative error {rel.max():.2e}"


def floor_act(x, act):
    """Largest value of the activation dtype that is <= x (x in fp64)."""
    x = np.asarray(x, dtype=np.float64)
    f = x.astype(np.float32)
    f = np.where(f.astype(np.float64) > x, np.nextafter(f, np.float32(-np.inf)), f)
    f = np.asarray(f, dtype=np.float32)
    if act == "f32":
        return f.astype(np.float64)
    bits = f.view(np.uint32)
    t = bits & np.uint32(0xFFFF0000)             # bf16 truncation (toward zero)
    t = np.where((f < 0) & (t != bits), t + np.uint32(0x10000), t).astype(np.uint32)
    return t.view(np.float32).astype(np.float64)


def ceil_act(x, act):
    return -floor_act(-np.asarray(x, dtype=np.float64), act)


def check_attention(got, ref, act, what=""):
    """The literal bound on the unrounded result: `got` (in the activation
    dtype) must be a rounding, up or down, of some value within atol of the
    fp64 oracle, i.e. lie between the dtype's neighbours of ref - atol and
    ref + atol.  atol is 2e-2 for bf16 and 1e-4 for fp32 outputs."""
    atol = 1e-4 if act == "f32" else 2e-2
    lo, hi = floor_act(ref - atol, act), ceil_act(ref + atol, act)
    bad = (got < lo) | (got > hi)
    if bad.any():
        i = np.unravel_index(int(np.argmax(np.abs(got - ref))), got.shape)
        raise AssertionError(f"{what}: {int(bad.sum())} outputs outside the bound; worst "
                             f"{got[i]:.6g} vs oracle {ref[i]:.6g} at {tuple(int(j) for j in i)}")
