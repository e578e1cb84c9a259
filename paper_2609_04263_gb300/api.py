"""PyTorch-facing wrappers over the C ABI: device memory and streams come from
torch, every computation runs in libkvq.so."""
from __future__ import annotations

import math

import torch

from . import kvq

_DT = {torch.float32: kvq.KVQ_F32, torch.bfloat16: kvq.KVQ_BF16}
_TORCH = {kvq.KVQ_F32: torch.float32, kvq.KVQ_BF16: torch.bfloat16}
_PLANE_DTYPE = {1: torch.uint8, 2: torch.float16, 4: torch.float32}


def _stream() -> int:
    return torch.cuda.current_stream().cuda_stream


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("tensor arguments must be contiguous CUDA tensors")
    return t.data_ptr()


def make_desc(fmt, key_bits, value_bits, group_size, batch, kv_heads, q_heads, head_dim,
              max_tokens, dtype, residual_tokens=0, sink_tokens=0, norm_iters=8,
              layout=kvq.KVQ_LAYOUT_UNIFORM, num_pages=0):
    return kvq.kvq_cache_desc(fmt=fmt, key_bits=key_bits, value_bits=value_bits,
                              group_size=group_size, residual_tokens=residual_tokens,
                              sink_tokens=sink_tokens, norm_iters=norm_iters, batch=batch,
                              kv_heads=kv_heads, q_heads=q_heads, head_dim=head_dim,
                              max_tokens=max_tokens, dtype=_DT.get(dtype, dtype),
                              layout=layout, num_pages=num_pages)


class Cache:
    """One layer's packed cache in a torch-owned device buffer."""

    def __init__(self, desc: kvq.kvq_cache_desc, device="cuda", buffer=None):
        self.desc = desc
        self.nbytes = kvq.kvq_cache_bytes(desc)
        if buffer is None:
            buffer = torch.empty(self.nbytes, dtype=torch.uint8, device=device)
        self.buffer = buffer
        self.handle = kvq.kvq_create_cache(desc, buffer.data_ptr(), self.nbytes)
        self.act = _TORCH[desc.dtype]

    def __del__(self):
        h = getattr(self, "handle", None)
        if h:
            kvq.kvq_destroy_cache(h)
            self.handle = None

    @property
    def tokens(self) -> int:
        return kvq.kvq_cache_tokens(self.handle)

    def reset(self) -> None:
        kvq.kvq_reset_cache(self.handle)

    def sync(self) -> int:
        """Refresh the host token count from the device (after graph replays)."""
        kvq.kvq_cache_sync(self.handle, _stream())
        return self.tokens

    def append(self, k: torch.Tensor, v: torch.Tensor) -> None:
        kvq.kvq_append_pack(self.handle, _ptr(k), _ptr(v), k.shape[2], _stream())

    def attend_prefill(self, q: torch.Tensor, out=None, scale=None) -> torch.Tensor:
        out = torch.empty_like(q) if out is None else out
        scale = 1.0 / math.sqrt(self.desc.head_dim) if scale is None else scale
        kvq.kvq_attend_prefill(self.handle, _ptr(q), q.shape[2], q.shape[1], scale, _ptr(out),
                               _stream())
        return out

    def attend_decode(self, q: torch.Tensor, out=None, scale=None) -> torch.Tensor:
        out = torch.empty_like(q) if out is None else out
        scale = 1.0 / math.sqrt(self.desc.head_dim) if scale is None else scale
        kvq.kvq_attend_decode(self.handle, _ptr(q), q.shape[1], scale, _ptr(out), _stream())
        return out

    def decode_step(self, x, w_qkv, lora, alpha_over_r, rope_base, qkv=None, out=None,
                    scale=None):
        """Project the new token x [B,1,d_in], append its key/value and attend:
        returns (q, k, v), out."""
        d = self.desc
        B, D = d.batch, d.head_dim
        if qkv is None:
            qkv = (torch.empty(B, d.q_heads, 1, D, dtype=x.dtype, device=x.device),
                   torch.empty(B, d.kv_heads, 1, D, dtype=x.dtype, device=x.device),
                   torch.empty(B, d.kv_heads, 1, D, dtype=x.dtype, device=x.device))
        out = torch.empty(B, d.q_heads, 1, D, dtype=x.dtype, device=x.device) if out is None else out
        scale = 1.0 / math.sqrt(D) if scale is None else scale
        args = []
        for p in "qkv":
            ab = lora.get(p)
            args += [None, None, 0] if ab is None else [_ptr(ab[0]), _ptr(ab[1]), ab[0].shape[0]]
        kvq.kvq_decode_step(self.handle, _ptr(x), x.shape[-1], _ptr(w_qkv), *args, alpha_over_r,
                            rope_base, scale, _ptr(qkv[0]), _ptr(qkv[1]), _ptr(qkv[2]), _ptr(out),
                            _stream())
        return qkv, out

    def project_append(self, x, w_qkv, lora, alpha_over_r, rope_base, q=None):
        """Project x [B,L,d_in] and code the new keys and values straight into
        the cache (positions continue it); returns q [B,Hq,L,D]."""
        d = self.desc
        B, L, d_in = x.shape
        q = torch.empty(B, d.q_heads, L, d.head_dim, dtype=x.dtype, device=x.device) if q is None else q
        args = []
        for p in "qkv":
            ab = lora.get(p)
            args += [None, None, 0] if ab is None else [_ptr(ab[0]), _ptr(ab[1]), ab[0].shape[0]]
        kvq.kvq_project_append(self.handle, _ptr(x), L, d_in, _ptr(w_qkv), *args, alpha_over_r,
                               rope_base, _ptr(q), _stream())
        return q

    def project_append_supported(self, L, d_in, lora) -> bool:
        r = [0 if lora.get(p) is None else lora[p][0].shape[0] for p in "qkv"]
        return kvq.kvq_project_append_supported(self.handle, L, d_in, *r)

    def decode_step_fused(self, d_in, lora) -> bool:
        """Whether decode_step with this d_in and these LoRA factors runs as
        one fused kernel."""
        r = [0 if lora.get(p) is None else lora[p][0].shape[0] for p in "qkv"]
        return kvq.kvq_decode_step_fused(self.handle, d_in, *r)

    def append_ragged(self, k, v, n=None) -> None:
        """Ragged / paged caches: sequence b appends the first n[b] of its
        rows of k, v [B, H, L, D] (all L when n is None)."""
        kvq.kvq_append_pack_ragged(self.handle, _ptr(k), _ptr(v), k.shape[2], n, _stream())

    def seq_tokens(self, b) -> int:
        return kvq.kvq_seq_tokens(self.handle, b)

    def seq_release(self, b) -> None:
        kvq.kvq_seq_release(self.handle, b, _stream())

    def free_pages(self) -> int:
        return kvq.kvq_free_pages(self.handle)

    def seq_pages(self, b) -> list:
        return kvq.kvq_seq_pages(self.handle, b)

    def attend_backward(self, q, d_out, scale=None, workspace=None):
        """Straight-through backward of attend_prefill(q): returns fp32
        (d_q [B,Hq,L,D], d_k, d_v [B,Hkv,T,D]), the gradients at the stored
        reconstruction, which by the estimator are those of the coded keys
        and values.  workspace: a uint8 device tensor (default: all pairs in
        one pass)."""
        d = self.desc
        B, Hq, L, D = q.shape
        T = self.tokens
        per = kvq.kvq_attend_backward_workspace(self.handle, L, Hq)
        if workspace is None:
            workspace = torch.empty(per * B * d.kv_heads, dtype=torch.uint8, device=q.device)
        scale = 1.0 / math.sqrt(D) if scale is None else scale
        f32 = dict(dtype=torch.float32, device=q.device)
        dq = torch.empty(B, Hq, L, D, **f32)
        dk = torch.empty(B, d.kv_heads, T, D, **f32)
        dv = torch.empty(B, d.kv_heads, T, D, **f32)
        kvq.kvq_attend_backward(self.handle, _ptr(q), _ptr(d_out), L, Hq, scale, _ptr(dq),
                                _ptr(dk), _ptr(dv), _ptr(workspace), workspace.numel(), _stream())
        return dq, dk, dv

    def planes(self) -> dict:
        """name -> tensor view [B, H, rows, cols] of each present plane."""
        v = kvq.kvq_cache_view(self.handle)
        base = self.buffer.data_ptr()
        out = {}
        for i, name in enumerate(kvq.PLANES):
            p = v.ptr[i]
            if not p:
                continue
            dims = [int(d) for d in v.dims[i]]
            eb = int(v.elem_bytes[i])
            n = dims[0] * dims[1] * dims[2] * dims[3] * eb
            off = p - base
            raw = self.buffer[off:off + n]
            dt = _PLANE_DTYPE[eb]
            if name.endswith(("_full", "_pend")):
                dt = self.act
            out[name] = raw.view(dt).view(*dims)
        out["_tokens"] = int(v.tokens)
        out["_quantized_tokens"] = int(v.quantized_tokens)
        return out


def project_lora(x, w_qkv, lora, alpha_over_r, n_q_heads, n_kv_heads, head_dim, pos0=0,
                 rope_base=0.0, out=None, pos_cache: "Cache | None" = None):
    """q [B,Hq,L,D], k, v [B,Hkv,L,D] = RoPE(x W'^T) with W' = W + (alpha/r) B A.

    lora: dict p -> (A [r, d_in], B [d_out, r]) or None for p in 'qkv'.
    Positions are pos0 + l, plus pos_cache's device token count if given.
    """
    B, L, d_in = x.shape
    D = head_dim
    if out is None:
        out = (torch.empty(B, n_q_heads, L, D, dtype=x.dtype, device=x.device),
               torch.empty(B, n_kv_heads, L, D, dtype=x.dtype, device=x.device),
               torch.empty(B, n_kv_heads, L, D, dtype=x.dtype, device=x.device))
    args = []
    for p in "qkv":
        ab = lora.get(p)
        if ab is None:
            args += [None, None, 0]
        else:
            args += [_ptr(ab[0]), _ptr(ab[1]), ab[0].shape[0]]
    kvq.kvq_project_lora(_ptr(x), B, L, d_in, _ptr(w_qkv), *args, alpha_over_r, n_q_heads,
                         n_kv_heads, head_dim, pos0,
                         pos_cache.handle if pos_cache is not None else None, rope_base,
                         _DT[x.dtype], _ptr(out[0]),
                         _ptr(out[1]), _ptr(out[2]), _stream())
    return out


def project_lora_nf4(x, w_codes, w_absmax, lora, alpha_over_r, n_q_heads, n_kv_heads, head_dim,
                     pos0=0, rope_base=0.0, out=None, pos_cache: "Cache | None" = None):
    """project_lora over an NF4 base: w_codes uint8 [N, d_in/2], w_absmax
    float32 [N, d_in/64]; the LoRA branches stay explicit bf16."""
    B, L, d_in = x.shape
    D = head_dim
    if out is None:
        out = (torch.empty(B, n_q_heads, L, D, dtype=x.dtype, device=x.device),
               torch.empty(B, n_kv_heads, L, D, dtype=x.dtype, device=x.device),
               torch.empty(B, n_kv_heads, L, D, dtype=x.dtype, device=x.device))
    args = []
    for p in "qkv":
        ab = lora.get(p)
        args += [None, None, 0] if ab is None else [_ptr(ab[0]), _ptr(ab[1]), ab[0].shape[0]]
    kvq.kvq_project_lora_nf4(_ptr(x), B, L, d_in, _ptr(w_codes), _ptr(w_absmax), *args,
                             alpha_over_r, n_q_heads, n_kv_heads, head_dim, pos0,
                             pos_cache.handle if pos_cache is not None else None, rope_base,
                             _ptr(out[0]), _ptr(out[1]), _ptr(out[2]), _stream())
    return out


def lora_backward(x, w_qkv, lora, alpha_over_r, n_q_heads, n_kv_heads, head_dim, d_q, d_k, d_v,
                  pos0=0, rope_base=0.0, want_dx=False, workspace=None):
    """Gradients of the rank-r factors of project_lora given fp32 gradients of
    its outputs (d_q [B,Hq,L,D]; d_k, d_v [B,Hkv,kv_rows,D], the last L rows
    belonging to x's tokens).  Returns ({p: (dA_p, dB_p) or None}, d_x or None),
    fp32; the base weight stays frozen (w_qkv is read only for d_x)."""
    B, L, d_in = x.shape
    D = head_dim
    r = [0 if lora.get(p) is None else lora[p][0].shape[0] for p in "qkv"]
    if workspace is None:
        nb = kvq.kvq_lora_backward_workspace(B, L, d_in, n_q_heads, n_kv_heads, D, *r)
        workspace = torch.empty(nb, dtype=torch.uint8, device=x.device)
    f32 = dict(dtype=torch.float32, device=x.device)
    grads, args = {}, []
    for i, p in enumerate("qkv"):
        ab = lora.get(p)
        if ab is None:
            grads[p] = None
            args += [None, None, 0]
        else:
            grads[p] = (torch.empty(ab[0].shape, **f32), torch.empty(ab[1].shape, **f32))
            args += [_ptr(ab[0]), _ptr(ab[1]), r[i]]
    gp = [None if grads[p] is None else _ptr(t) for p in "qkv" for t in (grads[p] or (None, None))]
    dx = torch.empty(B, L, d_in, **f32) if want_dx else None
    kvq.kvq_lora_backward(_ptr(x), B, L, d_in, _ptr(w_qkv), *args, alpha_over_r, n_q_heads,
                          n_kv_heads, D, pos0, rope_base, _DT[x.dtype], _ptr(d_q), _ptr(d_k),
                          _ptr(d_v), d_k.shape[2], *gp, _ptr(dx), _ptr(workspace),
                          workspace.numel(), _stream())
    return grads, dx

