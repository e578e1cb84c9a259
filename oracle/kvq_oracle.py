"""CPU oracle for the packed-cache attention step (test infrastructure only).

Only the tests, the smoke check and the benchmark's CPU-baseline leg may import
this module.  The library never calls it, and it shares no code with the CUDA
path: it is a plain, slow restatement of what the paper defines, written so a
reader can check it against the paper line by line.

Precision.  Everything that decides an integer (group minimum/maximum, scale,
code, the Hadamard butterflies and the dual-axis normalisation that precede a
code) is computed in IEEE fp32 in a fixed order, exactly as the cache format
fixes it, so packed bytes and fp16 metadata can be compared bit for bit.
Projections, reconstructions and attention are computed in fp64.

What each function follows (paper sections and equations):
  * projections            Section 3, Eq. (1)  Q = H W_Q^T, K = H W_K^T, V = H W_V^T
  * LoRA update            Section 3, Eq. (lora)  W' = W + (alpha/r) B A
  * adapter cost           Section 3.4: r (d_in + d_out) parameters / MACs per token
  * NF4 base weights       Section 2 (QLoRA's 4-bit NormalFloat), Sections 3.4 and
                           4 (NF4 bases with explicit adapters): levels, blocks of 64
                           inputs with one absmax each
  * affine quantizer       Section 3.1, Eq. (affine) + clipping to [0, 2^b - 1],
                           FP16 scale and FP16 offset
  * symmetric quantizer    Section 3.1: maximum-magnitude scale, no offset
  * physical cache         Section 3.1: new states packed and appended, no
                           unquantized copy kept (beyond the format's own
                           full-precision window)
  * KIVI K2V2              Sections 2 and 3.1: per-channel keys, per-token values,
                           group 32, 128-token full-precision residual
  * KVarN K4V2             Sections 2 and 3.1: protected sink tokens, fixed
                           normalised Hadamard, dual-axis variance normalisation
  * reconstruction R_phi   Section 3.2: attention sees the stored reconstruction
  * attention              Section 3.3: forward attention over the reconstruction
  * STE backward           Section 3.3: x_hat + x - stopgrad(x) for appended states;
                           attention and adapter gradients by fp64 autograd

Readings where the paper is silent are listed in the design notes (group
arithmetic order, code range of the symmetric quantizer, bit order, KIVI flush
rule, KVarN staging and normalisation details, RoPE convention).

Parity pins: every function here is pinned by the not-gpu tests against closed
forms, library routines, invariants or values the paper prints, except that the
KVarN format is pinned only by invariants and special cases (the official KVarN
code is not available), and end-to-end perplexity is out of reach (no weights
or data).
"""
from __future__ import annotations

import math

import numpy as np
import torch

F32 = np.float32
EPS = F32(1e-8)          # the scale floor of Eq. (affine)

FMT_FLOAT, FMT_AFFINE, FMT_SYMMETRIC, FMT_KIVI, FMT_KVARN = range(5)


# ----------------------------------------------------------------------------
# Activation dtype rounding (inputs and outputs of the path are bf16 or fp32)
# ----------------------------------------------------------------------------
def round_to(x, act: str) -> np.ndarray:
    """Round values to the activation dtype; returns float32 holding them.

    fp64 inputs are rounded to fp32 first (the kernels accumulate in fp32).
    """
    x32 = np.asarray(x, dtype=np.float32)
    if act == "f32":
        return x32
    if act == "bf16":
        return torch.from_numpy(np.ascontiguousarray(x32)).to(torch.bfloat16).to(
            torch.float32).numpy()
    raise ValueError(act)


# ----------------------------------------------------------------------------
# Section 3, Eq. (1) and Eq. (lora): LoRA-adapted Q/K/V projections, then RoPE
# ----------------------------------------------------------------------------
def rope_rotate_half(y: np.ndarray, pos: np.ndarray, base: float) -> np.ndarray:
    """Rotary position embedding, rotate-half convention, fp64.

    y [..., L, D]; pos [L] absolute positions.  Frequency i < D/2 is
    base^(-2i/D); channel i pairs with channel i + D/2.
    """
    D = y.shape[-1]
    half = D // 2
    i = np.arange(half, dtype=np.float64)
    theta = base ** (-2.0 * i / D)
    ang = pos.astype(np.float64)[:, None] * theta[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = y[..., :half], y[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def project_lora(x, w_qkv, lora, alpha_over_r, n_q_heads, n_kv_heads, head_dim,
                 pos0=0, rope_base=0.0):
    """Q, K, V for one layer in fp64, head-major [B, H, L, D].

    x [B, L, d_in]; w_qkv [(Hq + 2 Hkv) D, d_in] with Q rows, then K, then V;
    lora[p] = (A [r, d_in], B [d_out, r]) or None for p in 'qkv'.
    The adapter is the explicit branch (alpha/r) (x A^T) B^T, which equals
    x ((alpha/r) B A)^T, i.e. the projection by W' = W + (alpha/r) B A.
    RoPE (rope_base > 0) is applied to Q and K at positions pos0 + l.
    """
    x64 = np.asarray(x, dtype=np.float64)
    B, L, _ = x64.shape
    D = head_dim
    bounds = {"q": (0, n_q_heads * D),
              "k": (n_q_heads * D, (n_q_heads + n_kv_heads) * D),
              "v": ((n_q_heads + n_kv_heads) * D, (n_q_heads + 2 * n_kv_heads) * D)}
    heads = {"q": n_q_heads, "k": n_kv_heads, "v": n_kv_heads}
    pos = pos0 + np.arange(L)
    out = []
    for p in "qkv":
        lo, hi = bounds[p]
        w = np.asarray(w_qkv[lo:hi], dtype=np.float64)
        y = x64 @ w.T                                    # Eq. (1)
        if lora.get(p) is not None:
            a, b = (np.asarray(t, dtype=np.float64) for t in lora[p])
            y = y + alpha_over_r * ((x64 @ a.T) @ b.T)   # Eq. (lora), explicit
        y = y.reshape(B, L, heads[p], D).transpose(0, 2, 1, 3)
        if p in "qk" and rope_base > 0:
            y = rope_rotate_half(y, pos, rope_base)
        out.append(y)
    return tuple(out)


# ----------------------------------------------------------------------------
# NF4 base weights (Section 2 cites QLoRA's 4-bit NormalFloat for frozen bases;
# Sections 3.4 and 4 report NF4 Gemma and Llama-3.1 bases with explicit
# adapters).  A row of W is stored as 4-bit codes, one absmax scale per block
# of 64 consecutive inputs; a weight is level[code] * absmax.
# ----------------------------------------------------------------------------
NF4_BLOCK = 64


def nf4_levels() -> np.ndarray:
    """The 16 NF4 levels in fp64, built as QLoRA defines the data type:
    quantiles of the standard normal distribution, 8 for the positive half and
    7 for the negative half (so that zero is represented exactly), taken at
    evenly spaced probabilities from 1 - delta to 1/2 with
    delta = (1/30 + 1/32) / 2, then scaled so that the largest magnitude is 1."""
    from scipy.stats import norm     # the inverse normal CDF (library routine)
    delta = 0.5 * (1.0 / 30.0 + 1.0 / 32.0)
    pos = norm.ppf(np.linspace(1.0 - delta, 0.5, 9)[:-1])
    neg = -norm.ppf(np.linspace(1.0 - delta, 0.5, 8)[:-1])
    v = np.sort(np.concatenate([pos, [0.0], neg]))
    return v / np.abs(v).max()


def nf4_dequant(codes, absmax) -> np.ndarray:
    """W [N, d_in] in fp64 from codes [N, d_in / 2] (uint8; input k in byte
    k // 2, the low nibble for even k) and absmax [N, d_in / 64]."""
    codes = np.asarray(codes, dtype=np.uint8)
    idx = np.empty((codes.shape[0], codes.shape[1] * 2), dtype=np.int64)
    idx[:, 0::2] = codes & 0xF
    idx[:, 1::2] = codes >> 4
    w = nf4_levels()[idx]
    scale = np.repeat(np.asarray(absmax, dtype=np.float64), NF4_BLOCK, axis=1)
    return w * scale


def project_lora_nf4(x, codes, absmax, lora, alpha_over_r, n_q_heads, n_kv_heads, head_dim,
                     pos0=0, rope_base=0.0):
    """project_lora with the frozen base W_qkv given in NF4: the base weights
    are the dequantized ones, the rank-r branches stay explicit."""
    return project_lora(x, nf4_dequant(codes, absmax), lora, alpha_over_r, n_q_heads,
                        n_kv_heads, head_dim, pos0=pos0, rope_base=rope_base)


def adapter_params(d_in: int, d_out: int, r: int) -> int:
    """Section 3.4: an explicit rank-r adapter on W [d_out, d_in] adds
    r (d_in + d_out) parameters, and as many MACs per processed token."""
    return r * (d_in + d_out)


# ----------------------------------------------------------------------------
# Section 3.1, Eq. (affine): grouped quantizers, fp32, groups on the last axis
# ----------------------------------------------------------------------------
def affine_quant(x: np.ndarray, bits: int):
    """Eq. (affine) on groups laid along the last axis of x (fp32).

    s = max((max - min) / (2^b - 1), 1e-8); c = round((x - min) / s) with
    round-half-to-even, clipped to [0, 2^b - 1].  Codes use the fp32 s and
    min; the stored metadata are fp16(s) and fp16(min) (min + 0 so that -0 is
    stored as +0).  Returns (codes uint8, scale fp16, offset fp16).
    """
    x = np.asarray(x, dtype=F32)
    qmax = F32(2 ** bits - 1)
    mn = x.min(axis=-1)
    mx = x.max(axis=-1)
    s = np.maximum((mx - mn) / qmax, EPS)
    c = np.rint((x - mn[..., None]) / s[..., None])
    c = np.clip(c, F32(0), qmax).astype(np.uint8)
    mn = mn + F32(0.0)
    return c, s.astype(np.float16), mn.astype(np.float16)


def symmetric_quant(x: np.ndarray, bits: int):
    """Symmetric control of Section 3.1: maximum-magnitude scale, no offset.

    qmax = 2^(b-1) - 1; s = max(absmax / qmax, 1e-8); q = round(x / s)
    clipped to [-qmax, qmax]; stored unsigned as u = q + 2^(b-1).
    Returns (codes uint8, scale fp16).
    """
    x = np.asarray(x, dtype=F32)
    qmax = F32(2 ** (bits - 1) - 1)
    amax = np.abs(x).max(axis=-1)
    s = np.maximum(amax / qmax, EPS)
    q = np.clip(np.rint(x / s[..., None]), -qmax, qmax)
    u = (q + F32(2 ** (bits - 1))).astype(np.uint8)
    return u, s.astype(np.float16)


def affine_dequant(codes, s16, m16) -> np.ndarray:
    """x_hat = c * s + m, with the stored fp16 metadata, in fp64."""
    return (codes.astype(np.float64) * s16.astype(np.float64)[..., None]
            + m16.astype(np.float64)[..., None])


def symmetric_dequant(codes, s16, bits) -> np.ndarray:
    return ((codes.astype(np.float64) - 2 ** (bits - 1))
            * s16.astype(np.float64)[..., None])


def pack_codes(codes: np.ndarray, bits: int) -> np.ndarray:
    """Bit-pack codes along the last axis, LSB first: element j goes to byte
    floor(j b / 8) at bit (j b) mod 8."""
    per = 8 // bits
    n = codes.shape[-1]
    c = codes.reshape(*codes.shape[:-1], n // per, per).astype(np.uint16)
    out = np.zeros(c.shape[:-1], dtype=np.uint16)
    for j in range(per):
        out |= c[..., j] << (j * bits)
    return out.astype(np.uint8)


def unpack_codes(packed: np.ndarray, bits: int) -> np.ndarray:
    per = 8 // bits
    mask = (1 << bits) - 1
    p = packed.astype(np.uint16)
    parts = [(p >> (j * bits)) & mask for j in range(per)]
    return np.stack(parts, axis=-1).reshape(*packed.shape[:-1],
                                            packed.shape[-1] * per).astype(np.uint8)


# ----------------------------------------------------------------------------
# KVarN (Sections 2 and 3.1): fixed normalised Hadamard + dual-axis variance
# normalisation, fp32 in a fixed order
# ----------------------------------------------------------------------------
def fwht_f32(x: np.ndarray) -> np.ndarray:
    """Normalised Walsh-Hadamard transform (Sylvester order) on the last axis.

    Butterfly stages h = 1, 2, 4, ..., D/2 in that order, each mapping the pair
    (y[i], y[i+h]) to (y[i] + y[i+h], y[i] - y[i+h]) in fp32, then one
    multiply by fp32(1/sqrt(D)).  D must be a power of two.
    """
    y = np.array(x, dtype=F32)
    D = y.shape[-1]
    lead = y.shape[:-1]
    h = 1
    while h < D:
        v = y.reshape(*lead, D // (2 * h), 2, h)
        a, b = v[..., 0, :], v[..., 1, :]
        y = np.stack([a + b, a - b], axis=-2).reshape(*lead, D)
        h *= 2
    return y * F32(1.0 / math.sqrt(D))


def hadamard_matrix(D: int) -> np.ndarray:
    """The same normalised Sylvester matrix in fp64 (symmetric, orthogonal)."""
    H = np.ones((1, 1))
    while H.shape[0] < D:
        H = np.block([[H, H], [H, -H]])
    return H / math.sqrt(D)


def tree_sum_f32(a: np.ndarray) -> np.ndarray:
    """Sum over the last axis by the stride-halving pairwise tree in fp32:
    a[i] += a[i + n/2], then n /= 2, until one element is left."""
    a = np.array(a, dtype=F32)
    n = a.shape[-1]
    while n > 1:
        n //= 2
        a = a[..., :n] + a[..., n:2 * n]
    return a[..., 0]


def davn_f32(y: np.ndarray, iters: int):
    """Dual-axis variance normalisation of one block y [G tokens, D] (fp32).

    Each iteration divides every row by its RMS, then every column by its
    RMS, accumulating the divisors into row scales r [G] and column scales
    c [D] (so y_in = r_i c_j y_out up to rounding).  RMS floors at 1e-8.
    """
    y = np.array(y, dtype=F32)
    G, D = y.shape
    r = np.ones(G, dtype=F32)
    c = np.ones(D, dtype=F32)
    inv_d, inv_g = F32(1.0 / D), F32(1.0 / G)
    for _ in range(iters):
        sig = np.maximum(np.sqrt(tree_sum_f32(y * y) * inv_d), EPS)
        y = y / sig[:, None]
        r = r * sig
        sig = np.maximum(np.sqrt(tree_sum_f32((y * y).T) * inv_g), EPS)
        y = y / sig[None, :]
        c = c * sig
    return y, r, c


def kvarn_block_quant(x: np.ndarray, bits: int, group: int, iters: int,
                      rotate: bool = True):
    """One KVarN block x [G, D] -> (codes [G, D], s16 [G, D/g], m16 [G, D/g],
    r16 [G], c16 [D]).  Rotation, then normalisation, then grouped affine."""
    y = fwht_f32(x) if rotate else np.array(x, dtype=F32)
    y, r, c = davn_f32(y, iters)
    G, D = y.shape
    codes, s16, m16 = affine_quant(y.reshape(G, D // group, group), bits)
    return (codes.reshape(G, D), s16, m16, r.astype(np.float16),
            c.astype(np.float16))


def kvarn_block_dequant(codes, s16, m16, r16, c16, group, rotate=True):
    """Reconstruction of one block in fp64: r_i c_j (s c + m), rotated back."""
    G, D = codes.shape
    y = affine_dequant(codes.reshape(G, D // group, group), s16, m16).reshape(G, D)
    y = r16.astype(np.float64)[:, None] * c16.astype(np.float64)[None, :] * y
    if rotate:
        y = y @ hadamard_matrix(D)      # H is symmetric and its own inverse
    return y


# ----------------------------------------------------------------------------
# Section 3.1: the physical incremental cache
# ----------------------------------------------------------------------------
def kivi_quantized_prefix(T: int, residual: int, group: int) -> int:
    """Tokens of the KIVI cache held quantized once T tokens are stored:
    whole group-aligned blocks, keeping between R and R + group - 1 of the
    most recent tokens at full precision."""
    return group * (max(T - residual, 0) // group)


def kvarn_blocks(T: int, sinks: int, group: int) -> int:
    """Quantized KVarN blocks once T tokens are stored (after the sinks)."""
    return max(T - sinks, 0) // group


class OracleCache:
    """The cache of one layer, kept in exactly the byte layout the library
    uses, so that planes can be compared bit for bit.

    Planes (batch b, kv head h; codes are LSB-first bit-packed along D):
      FLOAT:          k_full, v_full [B,H,Tmax,D] (activation values)
      AFFINE / SYM:   k_codes [B,H,Tmax,D*kb/8], k_scale [B,H,Tmax,D/G] (fp16),
                      k_zero [B,H,Tmax,D/G] (affine only); same for v
      KIVI:           k_codes [B,H,Tmax,D*kb/8], k_scale/k_zero [B,H,Tmax/G,D]
                      (one group per 32-token block and channel); v_codes,
                      v_scale, v_zero per token as AFFINE; k_full/v_full is the
                      residual ring [B,H,R+G,D], token t in slot t mod (R+G)
      KVARN:          k_full/v_full are the sinks [B,H,S,D]; k_pend/v_pend the
                      staging ring [B,H,G,D] (slot (t-S) mod G); codes and
                      scale/zero per quantized token q = t - S as AFFINE,
                      k_row/v_row [B,H,Q] row scales, k_col/v_col [B,H,Q/G,D]
                      column scales (all fp16)
    """

    def __init__(self, fmt, key_bits, value_bits, group_size, batch, kv_heads,
                 head_dim, max_tokens, act="bf16", residual_tokens=0,
                 sink_tokens=0, norm_iters=8):
        self.fmt, self.kb, self.vb, self.G = fmt, key_bits, value_bits, group_size
        self.B, self.H, self.D, self.Tmax = batch, kv_heads, head_dim, max_tokens
        self.act, self.R, self.S, self.iters = act, residual_tokens, sink_tokens, norm_iters
        self.T = 0
        B, H, D, G, Tm = batch, kv_heads, head_dim, group_size, max_tokens
        f16, u8 = np.float16, np.uint8
        self.planes = {}
        P = self.planes
        if fmt == FMT_FLOAT:
            P["k_full"] = np.zeros((B, H, Tm, D), F32)
            P["v_full"] = np.zeros((B, H, Tm, D), F32)
        elif fmt in (FMT_AFFINE, FMT_SYMMETRIC):
            for n, b in (("k", key_bits), ("v", value_bits)):
                P[n + "_codes"] = np.zeros((B, H, Tm, D * b // 8), u8)
                P[n + "_scale"] = np.zeros((B, H, Tm, D // G), f16)
                if fmt == FMT_AFFINE:
                    P[n + "_zero"] = np.zeros((B, H, Tm, D // G), f16)
        elif fmt == FMT_KIVI:
            nblk = -(-Tm // G)
            P["k_codes"] = np.zeros((B, H, nblk * G, D * key_bits // 8), u8)
            P["k_scale"] = np.zeros((B, H, nblk, D), f16)
            P["k_zero"] = np.zeros((B, H, nblk, D), f16)
            P["v_codes"] = np.zeros((B, H, nblk * G, D * value_bits // 8), u8)
            P["v_scale"] = np.zeros((B, H, nblk * G, D // G), f16)
            P["v_zero"] = np.zeros((B, H, nblk * G, D // G), f16)
            P["k_full"] = np.zeros((B, H, self.R + G, D), F32)
            P["v_full"] = np.zeros((B, H, self.R + G, D), F32)
        elif fmt == FMT_KVARN:
            nblk = max(Tm - self.S, 0) // G
            Q = nblk * G
            P["k_full"] = np.zeros((B, H, self.S, D), F32)
            P["v_full"] = np.zeros((B, H, self.S, D), F32)
            P["k_pend"] = np.zeros((B, H, G, D), F32)
            P["v_pend"] = np.zeros((B, H, G, D), F32)
            for n, b in (("k", key_bits), ("v", value_bits)):
                P[n + "_codes"] = np.zeros((B, H, Q, D * b // 8), u8)
                P[n + "_scale"] = np.zeros((B, H, Q, D // G), f16)
                P[n + "_zero"] = np.zeros((B, H, Q, D // G), f16)
                P[n + "_row"] = np.zeros((B, H, Q), f16)
                P[n + "_col"] = np.zeros((B, H, nblk, D), f16)
        else:
            raise ValueError(fmt)

    # -- per-token grouped coding (AFFINE / SYMMETRIC, and KIVI values) ----
    def _code_tokens(self, name, x, bits, fmt, t0):
        """Code tokens x [B,H,n,D] into plane rows t0 .. t0+n-1."""
        B, H, n, D = x.shape
        G = self.G
        g = x.reshape(B, H, n, D // G, G)
        P = self.planes
        if fmt == FMT_SYMMETRIC:
            c, s = symmetric_quant(g, bits)
        else:
            c, s, m = affine_quant(g, bits)
            P[name + "_zero"][:, :, t0:t0 + n] = m
        P[name + "_scale"][:, :, t0:t0 + n] = s
        P[name + "_codes"][:, :, t0:t0 + n] = pack_codes(c.reshape(B, H, n, D), bits)

    def append(self, k, v):
        """Append L new tokens k, v [B, H, L, D] (activation-dtype values)."""
        k = np.asarray(k, dtype=F32)
        v = np.asarray(v, dtype=F32)
        L = k.shape[2]
        T0, T1 = self.T, self.T + L
        if T1 > self.Tmax:
            raise ValueError("cache capacity exceeded")
        P, G = self.planes, self.G
        if self.fmt == FMT_FLOAT:
            P["k_full"][:, :, T0:T1] = k
            P["v_full"][:, :, T0:T1] = v
        elif self.fmt in (FMT_AFFINE, FMT_SYMMETRIC):
            self._code_tokens("k", k, self.kb, self.fmt, T0)
            self._code_tokens("v", v, self.vb, self.fmt, T0)
        elif self.fmt == FMT_KIVI:
            ring = self.R + G
            q0 = kivi_quantized_prefix(T0, self.R, G)
            q1 = kivi_quantized_prefix(T1, self.R, G)

            def token(name, x, t):
                return x[:, :, t - T0] if t >= T0 else P[name + "_full"][:, :, t % ring]

            for blk0 in range(q0, q1, G):
                kb = np.stack([token("k", k, t) for t in range(blk0, blk0 + G)], axis=2)
                vb = np.stack([token("v", v, t) for t in range(blk0, blk0 + G)], axis=2)
                # keys: one group per channel over the block's G tokens
                c, s, m = affine_quant(kb.transpose(0, 1, 3, 2), self.kb)
                P["k_scale"][:, :, blk0 // G] = s
                P["k_zero"][:, :, blk0 // G] = m
                P["k_codes"][:, :, blk0:blk0 + G] = pack_codes(
                    c.transpose(0, 1, 3, 2), self.kb)
                # values: per token, groups of G along D
                self._code_tokens("v", vb, self.vb, FMT_AFFINE, blk0)
            for t in range(max(q1, T0), T1):
                P["k_full"][:, :, t % ring] = k[:, :, t - T0]
                P["v_full"][:, :, t % ring] = v[:, :, t - T0]
        elif self.fmt == FMT_KVARN:
            S = self.S
            for t in range(T0, min(S, T1)):
                P["k_full"][:, :, t] = k[:, :, t - T0]
                P["v_full"][:, :, t] = v[:, :, t - T0]
            n0, n1 = kvarn_blocks(T0, S, G), kvarn_blocks(T1, S, G)

            def token(name, x, t):
                return x[:, :, t - T0] if t >= T0 else P[name + "_pend"][:, :, (t - S) % G]

            for blk in range(n0, n1):
                ts = range(S + blk * G, S + (blk + 1) * G)
                for name, x, bits in (("k", k, self.kb), ("v", v, self.vb)):
                    xb = np.stack([token(name, x, t) for t in ts], axis=2)
                    for b in range(self.B):
                        for h in range(self.H):
                            c, s, m, r, cc = kvarn_block_quant(
                                xb[b, h], bits, G, self.iters)
                            rows = slice(blk * G, (blk + 1) * G)
                            P[name + "_codes"][b, h, rows] = pack_codes(c, bits)
                            P[name + "_scale"][b, h, rows] = s
                            P[name + "_zero"][b, h, rows] = m
                            P[name + "_row"][b, h, rows] = r
                            P[name + "_col"][b, h, blk] = cc
            for t in range(max(T0, S + n1 * G), T1):
                P["k_pend"][:, :, (t - S) % G] = k[:, :, t - T0]
                P["v_pend"][:, :, (t - S) % G] = v[:, :, t - T0]
        self.T = T1

    # -- Section 3.2: the reconstruction R_phi presented to attention ------
    def reconstruct(self):
        """K_hat, V_hat [B, H, T, D] in fp64 for every stored token."""
        P, G, T, D = self.planes, self.G, self.T, self.D
        B, H = self.B, self.H
        if self.fmt == FMT_FLOAT:
            return (P["k_full"][:, :, :T].astype(np.float64),
                    P["v_full"][:, :, :T].astype(np.float64))
        out = []
        for name, bits in (("k", self.kb), ("v", self.vb)):
            if self.fmt in (FMT_AFFINE, FMT_SYMMETRIC):
                c = unpack_codes(P[name + "_codes"][:, :, :T], bits).reshape(
                    B, H, T, D // G, G)
                s = P[name + "_scale"][:, :, :T]
                if self.fmt == FMT_AFFINE:
                    x = affine_dequant(c, s, P[name + "_zero"][:, :, :T])
                else:
                    x = symmetric_dequant(c, s, bits)
                out.append(x.reshape(B, H, T, D))
            elif self.fmt == FMT_KIVI:
                ring = self.R + G
                tq = kivi_quantized_prefix(T, self.R, G)
                x = np.zeros((B, H, T, D))
                c = unpack_codes(P[name + "_codes"][:, :, :tq], bits)
                if name == "k":
                    nb = tq // G
                    c = c.reshape(B, H, nb, G, D).transpose(0, 1, 2, 4, 3)
                    deq = affine_dequant(c, P["k_scale"][:, :, :nb], P["k_zero"][:, :, :nb])
                    x[:, :, :tq] = deq.transpose(0, 1, 2, 4, 3).reshape(B, H, tq, D)
                else:
                    c = c.reshape(B, H, tq, D // G, G)
                    deq = affine_dequant(c, P["v_scale"][:, :, :tq], P["v_zero"][:, :, :tq])
                    x[:, :, :tq] = deq.reshape(B, H, tq, D)
                for t in range(tq, T):
                    x[:, :, t] = P[name + "_full"][:, :, t % ring]
                out.append(x)
            else:  # KVARN
                S = self.S
                x = np.zeros((B, H, T, D))
                ns = min(S, T)
                x[:, :, :ns] = P[name + "_full"][:, :, :ns]
                nb = kvarn_blocks(T, S, G)
                c = unpack_codes(P[name + "_codes"][:, :, :nb * G], bits)
                for b in range(B):
                    for h in range(H):
                        for blk in range(nb):
                            rows = slice(blk * G, (blk + 1) * G)
                            x[b, h, S + blk * G:S + (blk + 1) * G] = kvarn_block_dequant(
                                c[b, h, rows], P[name + "_scale"][b, h, rows],
                                P[name + "_zero"][b, h, rows], P[name + "_row"][b, h, rows],
                                P[name + "_col"][b, h, blk], G)
                for t in range(S + nb * G, T):
                    x[:, :, t] = P[name + "_pend"][:, :, (t - S) % G]
                out.append(x)
        return tuple(out)


# ----------------------------------------------------------------------------
# Section 3.3: attention over the stored reconstruction
# ----------------------------------------------------------------------------
def attention(q, k_hat, v_hat, q_pos, scale):
    """softmax(q k_hat^T * scale + causal mask) v_hat in fp64.

    q [B, Hq, L, D]; k_hat, v_hat [B, Hkv, T, D]; query l sits at absolute
    position q_pos[l] and sees keys 0 .. q_pos[l].  Query head h reads kv head
    h // (Hq / Hkv).
    """
    q = np.asarray(q, dtype=np.float64)
    B, Hq, L, D = q.shape
    Hkv, T = k_hat.shape[1], k_hat.shape[2]
    g = Hq // Hkv
    kk = np.repeat(k_hat, g, axis=1)
    vv = np.repeat(v_hat, g, axis=1)
    s = np.einsum("bhld,bhtd->bhlt", q, kk) * scale
    visible = np.arange(T)[None, :] <= np.asarray(q_pos)[:, None]
    s = np.where(visible[None, None], s, -np.inf)
    s = s - s.max(axis=-1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=-1, keepdims=True)
    return np.einsum("bhlt,bhtd->bhld", p, vv)


def attend(cache: OracleCache, q, scale=None):
    """Attention of the L newest tokens' queries over the cache (the L tokens
    were appended last).  L = 1 is the decode step."""
    L = q.shape[2]
    k_hat, v_hat = cache.reconstruct()
    if scale is None:
        scale = 1.0 / math.sqrt(cache.D)
    return attention(q, k_hat, v_hat, np.arange(cache.T - L, cache.T), scale)


# ----------------------------------------------------------------------------
# Section 3.3: straight-through backward of the packed path.  Newly appended
# states are replaced by x_hat + x - stopgrad(x): the forward attention sees
# the stored reconstruction and the K and V adapters receive an identity
# backward path.  The gradients are taken by PyTorch autograd in fp64 (a
# library routine) through a torch restatement of attention() and
# project_lora() above; the tests pin both restatements to those functions.
# ----------------------------------------------------------------------------
def _attention_torch(q, k_hat, v_hat, q_pos, scale):
    B, Hq, L, D = q.shape
    Hkv, T = k_hat.shape[1], k_hat.shape[2]
    g = Hq // Hkv
    kk = k_hat.repeat_interleave(g, dim=1)
    vv = v_hat.repeat_interleave(g, dim=1)
    s = torch.einsum("bhld,bhtd->bhlt", q, kk) * scale
    visible = torch.arange(T)[None, :] <= torch.as_tensor(np.asarray(q_pos))[:, None]
    s = s.masked_fill(~visible[None, None], float("-inf"))
    p = torch.softmax(s, dim=-1)
    return torch.einsum("bhlt,bhtd->bhld", p, vv)


def attention_backward(q, k_hat, v_hat, q_pos, scale, d_out):
    """Gradients (dq, dk_hat, dv_hat) of sum(attention(q, k_hat, v_hat) * d_out)
    in fp64.  dk_hat, dv_hat [B, Hkv, T, D] collect every query head of the kv
    head's group.  By the straight-through estimator these are also the
    gradients of the keys and values that were coded into the cache."""
    t = lambda a: torch.tensor(np.asarray(a, dtype=np.float64), requires_grad=True)
    tq, tk, tv = t(q), t(k_hat), t(v_hat)
    o = _attention_torch(tq, tk, tv, q_pos, scale)
    (o * torch.as_tensor(np.asarray(d_out, dtype=np.float64))).sum().backward()
    return tq.grad.numpy(), tk.grad.numpy(), tv.grad.numpy()


def _rope_torch(y, pos, base):
    D = y.shape[-1]
    half = D // 2
    theta = base ** (-2.0 * torch.arange(half, dtype=torch.float64) / D)
    ang = torch.as_tensor(np.asarray(pos, dtype=np.float64))[:, None] * theta[None, :]
    c, s = torch.cos(ang), torch.sin(ang)
    x1, x2 = y[..., :half], y[..., half:]
    return torch.cat([x1 * c - x2 * s, x2 * c + x1 * s], dim=-1)


def _project_torch(x, w_qkv, lora_t, alpha_over_r, n_q_heads, n_kv_heads, head_dim, pos0,
                   rope_base):
    B, L, _ = x.shape
    D = head_dim
    bounds = {"q": (0, n_q_heads * D),
              "k": (n_q_heads * D, (n_q_heads + n_kv_heads) * D),
              "v": ((n_q_heads + n_kv_heads) * D, (n_q_heads + 2 * n_kv_heads) * D)}
    heads = {"q": n_q_heads, "k": n_kv_heads, "v": n_kv_heads}
    pos = pos0 + np.arange(L)
    out = []
    for p in "qkv":
        lo, hi = bounds[p]
        y = x @ w_qkv[lo:hi].T
        if lora_t.get(p) is not None:
            a, b = lora_t[p]
            y = y + alpha_over_r * ((x @ a.T) @ b.T)
        y = y.reshape(B, L, heads[p], D).transpose(1, 2)
        if p in "qk" and rope_base > 0:
            y = _rope_torch(y, pos, rope_base)
        out.append(y)
    return out


def lora_backward(x, w_qkv, lora, alpha_over_r, n_q_heads, n_kv_heads, head_dim, d_q, d_k,
                  d_v, pos0=0, rope_base=0.0):
    """Gradients of the rank-r factors, {p: (dA_p, dB_p)} in fp64, given the
    gradients d_q [B, Hq, L, D], d_k, d_v [B, Hkv, L, D] of the projection's
    outputs (q and k after RoPE) for the L tokens of x."""
    f64 = lambda a: torch.as_tensor(np.asarray(a, dtype=np.float64))
    lora_t = {}
    for p in "qkv":
        if lora.get(p) is None:
            lora_t[p] = None
        else:
            a, b = (f64(m).clone().requires_grad_(True) for m in lora[p])
            lora_t[p] = (a, b)
    q, k, v = _project_torch(f64(x), f64(w_qkv), lora_t, alpha_over_r, n_q_heads, n_kv_heads,
                             head_dim, pos0, rope_base)
    loss = (q * f64(d_q)).sum() + (k * f64(d_k)).sum() + (v * f64(d_v)).sum()
    leaves = [t for p in "qkv" if lora_t[p] is not None for t in lora_t[p]]
    if leaves:
        loss.backward()
    return {p: None if lora_t[p] is None else tuple(t.grad.numpy() for t in lora_t[p])
            for p in "qkv"}
