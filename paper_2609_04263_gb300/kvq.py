"""ctypes binding of libkvq.so: the same entry points as include/kvq.h.

Argument marshalling only.  Every step of the attention path runs in the
library's CUDA kernels; PyTorch provides device memory and streams.  The
library is loaded on first use and a missing build raises immediately.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libkvq.so")

KVQ_OK, KVQ_ERR_ARG, KVQ_ERR_SHAPE, KVQ_ERR_CAPACITY, KVQ_ERR_UNSUPPORTED, \
    KVQ_ERR_CUDA, KVQ_ERR_TIMEOUT = range(7)
KVQ_FMT_FLOAT, KVQ_FMT_AFFINE, KVQ_FMT_SYMMETRIC, KVQ_FMT_KIVI, KVQ_FMT_KVARN = range(5)
KVQ_F32, KVQ_BF16 = 0, 1
KVQ_LAYOUT_UNIFORM, KVQ_LAYOUT_RAGGED, KVQ_LAYOUT_PAGED = range(3)
KVQ_PAGE_TOKENS = 256
KVQ_MAX_SEQS = 512

PLANES = ["k_codes", "k_scale", "k_zero", "v_codes", "v_scale", "v_zero", "k_full",
          "v_full", "k_pend", "v_pend", "k_row", "k_col", "v_row", "v_col", "workspace"]
NUM_PLANES = len(PLANES)

c_int, c_float, c_void_p, c_size_t = ctypes.c_int, ctypes.c_float, ctypes.c_void_p, ctypes.c_size_t


class KvqError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"kvq status {status}: {msg}")
        self.status = status


class kvq_cache_desc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "fmt", "key_bits", "value_bits", "group_size", "residual_tokens", "sink_tokens",
        "norm_iters", "batch", "kv_heads", "q_heads", "head_dim", "max_tokens", "dtype",
        "layout", "num_pages")]


class kvq_cache_planes(ctypes.Structure):
    _fields_ = [("ptr", c_void_p * NUM_PLANES),
                ("dims", (ctypes.c_int64 * 4) * NUM_PLANES),
                ("elem_bytes", ctypes.c_int32 * NUM_PLANES),
                ("tokens", ctypes.c_int32),
                ("quantized_tokens", ctypes.c_int32)]


_SIGS = {
    "kvq_abi_version": (c_int, []),
    "kvq_last_error": (ctypes.c_char_p, []),
    "kvq_cache_bytes": (c_size_t, [ctypes.POINTER(kvq_cache_desc)]),
    "kvq_create_cache": (c_int, [ctypes.POINTER(kvq_cache_desc), c_void_p, c_size_t,
                                 ctypes.POINTER(c_void_p)]),
    "kvq_destroy_cache": (c_int, [c_void_p]),
    "kvq_reset_cache": (c_int, [c_void_p]),
    "kvq_cache_tokens": (c_int, [c_void_p]),
    "kvq_cache_view": (c_int, [c_void_p, ctypes.POINTER(kvq_cache_planes)]),
    "kvq_project_lora": (c_int, [c_void_p, c_int, c_int, c_int, c_void_p,
                                 c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_int,
                                 c_void_p, c_void_p, c_int, c_float, c_int, c_int, c_int,
                                 c_int, c_void_p, c_float, c_int, c_void_p, c_void_p, c_void_p,
                                 c_void_p]),
    "kvq_cache_sync": (c_int, [c_void_p, c_void_p]),
    "kvq_append_pack": (c_int, [c_void_p, c_void_p, c_void_p, c_int, c_void_p]),
    "kvq_attend_prefill": (c_int, [c_void_p, c_void_p, c_int, c_int, c_float, c_void_p,
                                   c_void_p]),
    "kvq_attend_decode": (c_int, [c_void_p, c_void_p, c_int, c_float, c_void_p, c_void_p]),
    "kvq_device_status": (c_int, [c_void_p, ctypes.POINTER(c_int)]),
    "kvq_attend_decode_noalloc": (c_int, [c_void_p, c_void_p, c_int, c_float, c_void_p,
                                          c_void_p]),
    "kvq_decode_step": (c_int, [c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_void_p, c_int,
                                c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_int, c_float,
                                c_float, c_float, c_void_p, c_void_p, c_void_p, c_void_p,
                                c_void_p]),
    "kvq_decode_step_fused": (c_int, [c_void_p, c_int, c_int, c_int, c_int]),
    "kvq_project_append": (c_int, [c_void_p, c_void_p, c_int, c_int, c_void_p, c_void_p, c_void_p,
                                   c_int, c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_int,
                                   c_float, c_float, c_void_p, c_void_p]),
    "kvq_project_append_supported": (c_int, [c_void_p, c_int, c_int, c_int, c_int, c_int]),
    "kvq_project_lora_nf4": (c_int, [c_void_p, c_int, c_int, c_int, c_void_p, c_void_p,
                                     c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_int,
                                     c_void_p, c_void_p, c_int, c_float, c_int, c_int, c_int,
                                     c_int, c_void_p, c_float, c_void_p, c_void_p, c_void_p,
                                     c_void_p]),
    "kvq_append_pack_ragged": (c_int, [c_void_p, c_void_p, c_void_p, c_int,
                                       ctypes.POINTER(c_int), c_void_p]),
    "kvq_seq_tokens": (c_int, [c_void_p, c_int]),
    "kvq_seq_release": (c_int, [c_void_p, c_int, c_void_p]),
    "kvq_free_pages": (c_int, [c_void_p]),
    "kvq_seq_pages": (c_int, [c_void_p, c_int, ctypes.POINTER(c_int), c_int]),
    "kvq_attend_backward_workspace": (c_size_t, [c_void_p, c_int, c_int]),
    "kvq_attend_backward": (c_int, [c_void_p, c_void_p, c_void_p, c_int, c_int, c_float,
                                    c_void_p, c_void_p, c_void_p, c_void_p, c_size_t,
                                    c_void_p]),
    "kvq_lora_backward_workspace": (c_size_t, [c_int, c_int, c_int, c_int, c_int, c_int, c_int,
                                               c_int, c_int]),
    "kvq_lora_backward": (c_int, [c_void_p, c_int, c_int, c_int, c_void_p,
                                  c_void_p, c_void_p, c_int, c_void_p, c_void_p, c_int,
                                  c_void_p, c_void_p, c_int, c_float, c_int, c_int, c_int,
                                  c_int, c_float, c_int, c_void_p, c_void_p, c_void_p, c_int,
                                  c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                  c_void_p, c_void_p, c_size_t, c_void_p]),
}

_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "paper_2609_04263_gb300.build.build()")
        so = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(so, name)
            fn.restype, fn.argtypes = res, args
        _lib = so
    return _lib


def _check(status: int) -> None:
    if status != KVQ_OK:
        raise KvqError(status, kvq_last_error())


def kvq_last_error() -> str:
    return lib().kvq_last_error().decode()


def kvq_abi_version() -> int:
    return lib().kvq_abi_version()


def kvq_cache_bytes(desc: kvq_cache_desc) -> int:
    n = lib().kvq_cache_bytes(ctypes.byref(desc))
    if n == 0:
        raise KvqError(KVQ_ERR_SHAPE, kvq_last_error())
    return n


def kvq_create_cache(desc: kvq_cache_desc, dev_buf: int, nbytes: int) -> int:
    out = c_void_p()
    _check(lib().kvq_create_cache(ctypes.byref(desc), c_void_p(dev_buf), nbytes,
                                  ctypes.byref(out)))
    return out.value


def kvq_destroy_cache(handle: int) -> None:
    _check(lib().kvq_destroy_cache(c_void_p(handle)))


def kvq_reset_cache(handle: int) -> None:
    _check(lib().kvq_reset_cache(c_void_p(handle)))


def kvq_cache_tokens(handle: int) -> int:
    return lib().kvq_cache_tokens(c_void_p(handle))


def kvq_cache_view(handle: int) -> kvq_cache_planes:
    out = kvq_cache_planes()
    _check(lib().kvq_cache_view(c_void_p(handle), ctypes.byref(out)))
    return out


def kvq_project_lora(x, B, L, d_in, w_qkv, a_q, b_q, r_q, a_k, b_k, r_k, a_v, b_v, r_v,
                     alpha_over_r, n_q_heads, n_kv_heads, head_dim, pos0, pos_cache,
                     rope_base, dtype, q, k, v, stream) -> None:
    P = lambda t: c_void_p(t or 0)
    _check(lib().kvq_project_lora(P(x), B, L, d_in, P(w_qkv), P(a_q), P(b_q), r_q, P(a_k),
                                  P(b_k), r_k, P(a_v), P(b_v), r_v, alpha_over_r, n_q_heads,
                                  n_kv_heads, head_dim, pos0, P(pos_cache), rope_base, dtype,
                                  P(q), P(k), P(v), P(stream)))


def kvq_cache_sync(handle, stream=0) -> None:
    _check(lib().kvq_cache_sync(c_void_p(handle), c_void_p(stream or 0)))


def kvq_append_pack(handle, k, v, L, stream) -> None:
    _check(lib().kvq_append_pack(c_void_p(handle), c_void_p(k), c_void_p(v), L,
                                 c_void_p(stream or 0)))


def kvq_attend_prefill(handle, q, L, n_q_heads, softmax_scale, out, stream) -> None:
    _check(lib().kvq_attend_prefill(c_void_p(handle), c_void_p(q), L, n_q_heads,
                                    softmax_scale, c_void_p(out), c_void_p(stream or 0)))


def kvq_attend_decode(handle, q, n_q_heads, softmax_scale, out, stream) -> None:
    _check(lib().kvq_attend_decode(c_void_p(handle), c_void_p(q), n_q_heads, softmax_scale,
                                   c_void_p(out), c_void_p(stream or 0)))


def kvq_attend_decode_noalloc(handle, q, n_q_heads, softmax_scale, out, stream) -> None:
    """Decode attention whose split-K partials live in the library's static
    device memory instead of the cache's workspace (nothing is allocated)."""
    _check(lib().kvq_attend_decode_noalloc(c_void_p(handle), c_void_p(q), n_q_heads,
                                           softmax_scale, c_void_p(out), c_void_p(stream or 0)))


def kvq_decode_step(handle, x, d_in, w_qkv, a_q, b_q, r_q, a_k, b_k, r_k, a_v, b_v, r_v,
                    alpha_over_r, rope_base, softmax_scale, q, k, v, out, stream) -> None:
    P = lambda t: c_void_p(t or 0)
    _check(lib().kvq_decode_step(c_void_p(handle), P(x), d_in, P(w_qkv), P(a_q), P(b_q), r_q,
                                 P(a_k), P(b_k), r_k, P(a_v), P(b_v), r_v, alpha_over_r,
                                 rope_base, softmax_scale, P(q), P(k), P(v), P(out), P(stream)))


def kvq_decode_step_fused(handle, d_in, r_q, r_k, r_v) -> bool:
    """True when kvq_decode_step with these shapes runs as one fused kernel."""
    return lib().kvq_decode_step_fused(c_void_p(handle), d_in, r_q, r_k, r_v) == 1


def kvq_device_status(stream=0) -> int:
    out = c_int(0)
    st = lib().kvq_device_status(c_void_p(stream or 0), ctypes.byref(out))
    if st not in (KVQ_OK, KVQ_ERR_TIMEOUT):
        _check(st)
    return out.value


def kvq_project_append(handle, x, L, d_in, w_qkv, a_q, b_q, r_q, a_k, b_k, r_k, a_v, b_v, r_v,
                       alpha_over_r, rope_base, q, stream=0) -> None:
    _check(lib().kvq_project_append(c_void_p(handle), c_void_p(x), L, d_in, c_void_p(w_qkv),
                                    c_void_p(a_q), c_void_p(b_q), r_q, c_void_p(a_k),
                                    c_void_p(b_k), r_k, c_void_p(a_v), c_void_p(b_v), r_v,
                                    alpha_over_r, rope_base, c_void_p(q), c_void_p(stream or 0)))


def kvq_project_append_supported(handle, L, d_in, r_q, r_k, r_v) -> bool:
    return lib().kvq_project_append_supported(c_void_p(handle), L, d_in, r_q, r_k, r_v) == 1


def kvq_project_lora_nf4(x, B, L, d_in, w_codes, w_absmax, a_q, b_q, r_q, a_k, b_k, r_k, a_v,
                         b_v, r_v, alpha_over_r, n_q_heads, n_kv_heads, head_dim, pos0,
                         pos_cache, rope_base, q, k, v, stream=0) -> None:
    _check(lib().kvq_project_lora_nf4(
        c_void_p(x), B, L, d_in, c_void_p(w_codes), c_void_p(w_absmax), c_void_p(a_q),
        c_void_p(b_q), r_q, c_void_p(a_k), c_void_p(b_k), r_k, c_void_p(a_v), c_void_p(b_v), r_v,
        alpha_over_r, n_q_heads, n_kv_heads, head_dim, pos0, c_void_p(pos_cache), rope_base,
        c_void_p(q), c_void_p(k), c_void_p(v), c_void_p(stream or 0)))


def kvq_attend_backward_workspace(handle, L, n_q_heads) -> int:
    return lib().kvq_attend_backward_workspace(c_void_p(handle), L, n_q_heads)


def kvq_attend_backward(handle, q, d_out, L, n_q_heads, softmax_scale, d_q, d_k, d_v,
                        workspace, workspace_bytes, stream=0) -> None:
    _check(lib().kvq_attend_backward(c_void_p(handle), c_void_p(q), c_void_p(d_out), L,
                                     n_q_heads, softmax_scale, c_void_p(d_q), c_void_p(d_k),
                                     c_void_p(d_v), c_void_p(workspace), workspace_bytes,
                                     c_void_p(stream or 0)))


def kvq_lora_backward_workspace(B, L, d_in, n_q_heads, n_kv_heads, head_dim, r_q, r_k,
                                r_v) -> int:
    return lib().kvq_lora_backward_workspace(B, L, d_in, n_q_heads, n_kv_heads, head_dim, r_q,
                                             r_k, r_v)


def kvq_lora_backward(x, B, L, d_in, w_qkv, a_q, b_q, r_q, a_k, b_k, r_k, a_v, b_v, r_v,
                      alpha_over_r, n_q_heads, n_kv_heads, head_dim, pos0, rope_base, dtype,
                      d_q, d_k, d_v, kv_rows, da_q, db_q, da_k, db_k, da_v, db_v, d_x,
                      workspace, workspace_bytes, stream=0) -> None:
    _check(lib().kvq_lora_backward(
        c_void_p(x), B, L, d_in, c_void_p(w_qkv), c_void_p(a_q), c_void_p(b_q), r_q,
        c_void_p(a_k), c_void_p(b_k), r_k, c_void_p(a_v), c_void_p(b_v), r_v, alpha_over_r,
        n_q_heads, n_kv_heads, head_dim, pos0, rope_base, dtype, c_void_p(d_q), c_void_p(d_k),
        c_void_p(d_v), kv_rows, c_void_p(da_q), c_void_p(db_q), c_void_p(da_k), c_void_p(db_k),
        c_void_p(da_v), c_void_p(db_v), c_void_p(d_x), c_void_p(workspace), workspace_bytes,
        c_void_p(stream or 0)))


def kvq_append_pack_ragged(handle, k, v, L, n=None, stream=0) -> None:
    arr = None if n is None else (c_int * len(n))(*[int(x) for x in n])
    _check(lib().kvq_append_pack_ragged(c_void_p(handle), c_void_p(k), c_void_p(v), L, arr,
                                        c_void_p(stream or 0)))


def kvq_seq_tokens(handle, b) -> int:
    return lib().kvq_seq_tokens(c_void_p(handle), b)


def kvq_seq_release(handle, b, stream=0) -> None:
    _check(lib().kvq_seq_release(c_void_p(handle), b, c_void_p(stream or 0)))


def kvq_free_pages(handle) -> int:
    return lib().kvq_free_pages(c_void_p(handle))


def kvq_seq_pages(handle, b) -> list:
    n = lib().kvq_seq_pages(c_void_p(handle), b, None, 0)
    if n < 0:
        return []
    buf = (c_int * max(n, 1))()
    lib().kvq_seq_pages(c_void_p(handle), b, buf, n)
    return [buf[i] for i in range(n)]

