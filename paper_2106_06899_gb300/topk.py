"""Thin ctypes binding of libtopk.so (include/topk_attention.h).

Argument marshalling only: every step of the computation runs in the CUDA
library.  Functions carry the C-ABI names; they take torch tensors, read
sizes from their shapes, pass raw pointers and raise ``TopkError`` on a
non-zero return code.  There is no fallback: if libtopk.so is missing or
no GB300 is present the calls fail loudly.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libtopk.so")

TOPK_F32, TOPK_BF16 = 0, 1
_lock = threading.Lock()
_lib = None


class TopkError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {error_string(code)} (code {code})")


def lib() -> ctypes.CDLL:
    """The loaded libtopk.so.  Raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise ImportError(f"{LIB_PATH} is not built; run `python -m paper_2106_06899_gb300.build` "
                                  "(nvcc for sm_103a) first")
            L = ctypes.CDLL(LIB_PATH)
            vp, i32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
            L.topk_attn_fwd.argtypes = [vp, vp, vp, vp] + [i32] * 9 + [vp]
            L.topk_attn_fwd_indices.argtypes = [vp, vp, vp, vp] + [i32] * 9 + [vp, vp, vp]
            L.topk_ffn_fwd.argtypes = [vp, vp, vp, vp] + [i32] * 4 + [vp]
            L.topk_ffn_fwd_indices.argtypes = [vp, vp, vp, vp] + [i32] * 4 + [vp, vp, vp]
            L.topk_attn_fwd_host.argtypes = [vp, vp, vp, vp] + [i32] * 9 + [vp]
            L.topk_ffn_fwd_host.argtypes = [vp, vp, vp, vp] + [i32] * 4 + [vp]
            L.topk_ffn_fwd_noalloc.argtypes = [vp, vp, vp, vp] + [i32] * 4 + [vp]
            L.topk_attn_workspace_bytes.argtypes = [i32] * 8
            L.topk_attn_workspace_bytes.restype = sz
            L.topk_ffn_workspace_bytes.argtypes = [i32] * 4
            L.topk_ffn_workspace_bytes.restype = sz
            L.topk_attn_fwd_masked.argtypes = [vp, vp, vp, vp] + [i32] * 8 + [vp, vp, ctypes.c_longlong,
                                                                            ctypes.c_longlong, i32, vp, vp, vp]
            L.topk_vanilla_attn_fwd.argtypes = [vp, vp, vp, vp] + [i32] * 7 + [vp, i32, vp]
            L.topk_vanilla_attn_workspace_bytes.argtypes = [i32] * 6
            L.topk_vanilla_attn_workspace_bytes.restype = sz
            L.topk_vanilla_ffn_fwd.argtypes = [vp, vp, vp, vp] + [i32] * 4 + [vp]
            L.topk_vanilla_ffn_workspace_bytes.argtypes = [i32] * 4
            L.topk_vanilla_ffn_workspace_bytes.restype = sz
            L.topk_attn_bwd.argtypes = [vp] * 9 + [i32] * 7 + [vp]
            L.topk_ffn_bwd.argtypes = [vp] * 9 + [i32] * 4 + [vp]
            L.topk_attn_bwd_workspace_bytes.argtypes = [i32] * 7
            L.topk_attn_bwd_workspace_bytes.restype = sz
            L.topk_ffn_bwd_workspace_bytes.argtypes = [i32] * 4
            L.topk_ffn_bwd_workspace_bytes.restype = sz
            L.topk_check.argtypes = [vp]
            L.topk_error_string.argtypes = [i32]
            L.topk_error_string.restype = ctypes.c_char_p
            L.topk_last_launch_count.argtypes = []
            L.topk_set_wait_limit_us.argtypes = [ctypes.c_longlong]
            L.topk_set_wait_limit_us.restype = ctypes.c_longlong
            L.topk_debug_skip_arrive.argtypes = [i32]
            L.topk_pool_usage.argtypes = [ctypes.POINTER(sz), ctypes.POINTER(sz), i32]
            L.topk_pool_trim.argtypes = []
            for f in ("topk_attn_fwd", "topk_attn_fwd_indices", "topk_ffn_fwd", "topk_ffn_fwd_indices",
                      "topk_attn_fwd_host", "topk_ffn_fwd_host", "topk_ffn_fwd_noalloc", "topk_check",
                      "topk_last_launch_count",
                      "topk_debug_skip_arrive", "topk_pool_usage", "topk_pool_trim", "topk_attn_bwd",
                      "topk_ffn_bwd", "topk_attn_fwd_masked", "topk_vanilla_attn_fwd", "topk_vanilla_ffn_fwd"):
                getattr(L, f).restype = i32
            _lib = L
    return _lib


def error_string(code: int) -> str:
    return lib().topk_error_string(int(code)).decode()


def _check(rc: int, where: str) -> None:
    if rc != 0:
        raise TopkError(rc, where)


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return TOPK_F32
    if t.dtype == torch.bfloat16:
        return TOPK_BF16
    raise TypeError(f"unsupported dtype {t.dtype}; use float32 or bfloat16")


def _ptr(t):
    return None if t is None else t.data_ptr()


def _attn_dims(q, k, v, out):
    for name, t in (("q", q), ("k", k), ("v", v), ("out", out)):
        if t.dim() != 4 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous [B, H, L, d] tensor")
    B, H, Lq, d = q.shape
    Lk = k.shape[2]
    if tuple(k.shape) != (B, H, Lk, d) or tuple(v.shape) != (B, H, Lk, d) or tuple(out.shape) != (B, H, Lq, d):
        raise ValueError("shape mismatch between q, k, v, out")
    if not (q.dtype == k.dtype == v.dtype == out.dtype):
        raise TypeError("q, k, v, out must share a dtype")
    return B, H, Lq, Lk, d


def topk_attn_fwd(q, k, v, out, topk: int, chunk: int = 1024, causal: bool = False, stream=None) -> None:
    """Eq. 4 top-k attention into ``out`` (device tensors [B,H,L,d], fp32 or bf16)."""
    B, H, Lq, Lk, d = _attn_dims(q, k, v, out)
    rc = lib().topk_attn_fwd(_ptr(q), _ptr(k), _ptr(v), _ptr(out), B, H, Lq, Lk, d, int(topk), int(chunk),
                             int(bool(causal)), _dtype_code(q), _stream(stream))
    _check(rc, "topk_attn_fwd")


def topk_attn_fwd_indices(q, k, v, out, topk: int, chunk: int = 1024, causal: bool = False, idx=None,
                          score=None, stream=None) -> None:
    """topk_attn_fwd plus kept indices idx [B,H,Lq,topk] int32 and scores [B,H,Lq,topk] fp32."""
    B, H, Lq, Lk, d = _attn_dims(q, k, v, out)
    for name, t, dt in (("idx", idx, torch.int32), ("score", score, torch.float32)):
        if t is not None and (t.dtype != dt or tuple(t.shape) != (B, H, Lq, topk) or not t.is_contiguous()):
            raise ValueError(f"{name} must be a contiguous [B,H,Lq,topk] {dt} tensor")
    rc = lib().topk_attn_fwd_indices(_ptr(q), _ptr(k), _ptr(v), _ptr(out), B, H, Lq, Lk, d, int(topk), int(chunk),
                                     int(bool(causal)), _dtype_code(q), _ptr(idx), _ptr(score), _stream(stream))
    _check(rc, "topk_attn_fwd_indices")


def pack_mask(mask: torch.Tensor):
    """A boolean mask [B or 1, H or 1, Lq, Lk] (True = the key takes part, Eq. 2's B_ij = 0) in the
    C ABI's layout: bit j % 32 of int32 word j // 32 of each query row, on mask's device.

    Returns (words [B|1, H|1, Lq, ceil(Lk/32)] int32, batch stride, head stride) in words; a stride is
    0 where the mask has one entry for all batches or heads."""
    if mask.dim() != 4 or mask.dtype != torch.bool:
        raise ValueError("mask must be a 4-D bool tensor [B or 1, H or 1, Lq, Lk]")
    mb, mh, Lq, Lk = mask.shape
    W = (Lk + 31) // 32
    padded = torch.zeros(mb, mh, Lq, W * 32, dtype=torch.int64, device=mask.device)
    padded[..., :Lk] = mask.to(torch.int64)
    shifts = torch.arange(32, dtype=torch.int64, device=mask.device)
    words = (padded.view(mb, mh, Lq, W, 32) << shifts).sum(dim=-1)
    words = torch.where(words >= 2**31, words - 2**32, words).to(torch.int32).contiguous()
    hs = Lq * W if mh > 1 else 0
    bs = mh * Lq * W if mb > 1 else 0
    return words, bs, hs


def topk_attn_fwd_masked(q, k, v, out, topk: int, chunk: int = 1024, causal: bool = False, kv_len=None,
                         mask_words=None, mask_batch_stride: int = 0, mask_head_stride: int = 0, idx=None,
                         score=None, stream=None) -> None:
    """Eq. 4 under Eq. 2's masks: causal (queries are the last Lq positions), kv_len [B] int32 (keys per
    batch) and a packed bit mask (see pack_mask); idx/score as topk_attn_fwd_indices, or None."""
    B, H, Lq, Lk, d = _attn_dims(q, k, v, out)
    if kv_len is not None and (kv_len.dtype != torch.int32 or tuple(kv_len.shape) != (B,)):
        raise ValueError("kv_len must be a [B] int32 tensor")
    if mask_words is not None:
        W = (Lk + 31) // 32
        if mask_words.dtype != torch.int32 or not mask_words.is_contiguous() or mask_words.shape[-2:] != (Lq, W):
            raise ValueError("mask_words must be a contiguous int32 [..., Lq, ceil(Lk/32)] tensor (pack_mask)")
    for name, t, dt in (("idx", idx, torch.int32), ("score", score, torch.float32)):
        if t is not None and (t.dtype != dt or tuple(t.shape) != (B, H, Lq, topk) or not t.is_contiguous()):
            raise ValueError(f"{name} must be a contiguous [B,H,Lq,topk] {dt} tensor")
    rc = lib().topk_attn_fwd_masked(_ptr(q), _ptr(k), _ptr(v), _ptr(out), B, H, Lq, Lk, d, int(topk), int(chunk),
                                    int(bool(causal)), _ptr(kv_len), _ptr(mask_words), int(mask_batch_stride),
                                    int(mask_head_stride), _dtype_code(q), _ptr(idx), _ptr(score), _stream(stream))
    _check(rc, "topk_attn_fwd_masked")


def topk_vanilla_attn_fwd(q, k, v, out, chunk: int = 1024, causal: bool = False, kv_len=None,
                          stream=None) -> None:
    """Plain attention (Eq. 1) over every valid key, the comparison path (bf16, d 64 or 128)."""
    B, H, Lq, Lk, d = _attn_dims(q, k, v, out)
    if kv_len is not None and (kv_len.dtype != torch.int32 or tuple(kv_len.shape) != (B,)):
        raise ValueError("kv_len must be a [B] int32 tensor")
    rc = lib().topk_vanilla_attn_fwd(_ptr(q), _ptr(k), _ptr(v), _ptr(out), B, H, Lq, Lk, d, int(chunk),
                                     int(bool(causal)), _ptr(kv_len), _dtype_code(q), _stream(stream))
    _check(rc, "topk_vanilla_attn_fwd")


def topk_vanilla_attn_workspace_bytes(B, H, Lq, Lk, d, dtype) -> int:
    return int(lib().topk_vanilla_attn_workspace_bytes(B, H, Lq, Lk, d, dtype))


def vanilla_attention(q, k, v, chunk: int = 1024, causal: bool = False, kv_len=None, stream=None):
    out = torch.empty_like(q)
    topk_vanilla_attn_fwd(q, k, v, out, chunk, causal, kv_len, stream)
    return out


def topk_vanilla_ffn_fwd(x, W1, W2, out, chunk: int = 16384, stream=None) -> None:
    """The dense FF layer (Eq. 3 without top-k) in d_ff slices of `chunk` keys: out fp32 [N, d_model]."""
    N, dm, dff = _ffn_dims(x, W1, W2, out)
    rc = lib().topk_vanilla_ffn_fwd(_ptr(x), _ptr(W1), _ptr(W2), _ptr(out), N, dm, dff, int(chunk), _stream(stream))
    _check(rc, "topk_vanilla_ffn_fwd")


def topk_vanilla_ffn_workspace_bytes(N, d_model, d_ff, chunk) -> int:
    return int(lib().topk_vanilla_ffn_workspace_bytes(N, d_model, d_ff, chunk))


def vanilla_ffn(x, W1, W2, chunk: int = 16384, stream=None):
    out = torch.empty(x.shape[0], x.shape[1], dtype=torch.float32, device=x.device)
    topk_vanilla_ffn_fwd(x, W1, W2, out, chunk, stream)
    return out


def topk_attn_fwd_host(q, k, v, out, topk: int, chunk: int = 1024, causal: bool = False, stream=None) -> None:
    """End-to-end call on HOST tensors (pinned is fastest); synchronises the stream."""
    B, H, Lq, Lk, d = _attn_dims(q, k, v, out)
    rc = lib().topk_attn_fwd_host(_ptr(q), _ptr(k), _ptr(v), _ptr(out), B, H, Lq, Lk, d, int(topk), int(chunk),
                                  int(bool(causal)), _dtype_code(q), _stream(stream))
    _check(rc, "topk_attn_fwd_host")


def _ffn_dims(x, W1, W2, out):
    for name, t in (("x", x), ("W1", W1), ("W2", W2), ("out", out)):
        if t.dim() != 2 or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous 2-D tensor")
    N, dm = x.shape
    dff = W1.shape[0]
    if tuple(W1.shape) != (dff, dm) or tuple(W2.shape) != (dff, dm) or tuple(out.shape) != (N, dm):
        raise ValueError("shape mismatch between x, W1, W2, out")
    if not (x.dtype == W1.dtype == W2.dtype == torch.bfloat16) or out.dtype != torch.float32:
        raise TypeError("x, W1, W2 must be bfloat16 and out float32")
    return N, dm, dff


def topk_ffn_fwd(x, W1, W2, out, topk: int, stream=None) -> None:
    """Eq. 3 with top-k: out [N, d_model] fp32 from x [N, d_model], W1/W2 [d_ff, d_model] bf16."""
    N, dm, dff = _ffn_dims(x, W1, W2, out)
    rc = lib().topk_ffn_fwd(_ptr(x), _ptr(W1), _ptr(W2), _ptr(out), N, dm, dff, int(topk), _stream(stream))
    _check(rc, "topk_ffn_fwd")


def topk_ffn_fwd_indices(x, W1, W2, out, topk: int, idx=None, score=None, stream=None) -> None:
    N, dm, dff = _ffn_dims(x, W1, W2, out)
    rc = lib().topk_ffn_fwd_indices(_ptr(x), _ptr(W1), _ptr(W2), _ptr(out), N, dm, dff, int(topk), _ptr(idx),
                                    _ptr(score), _stream(stream))
    _check(rc, "topk_ffn_fwd_indices")


def topk_ffn_fwd_host(x, W1, W2, out, topk: int, stream=None) -> None:
    N, dm, dff = _ffn_dims(x, W1, W2, out)
    rc = lib().topk_ffn_fwd_host(_ptr(x), _ptr(W1), _ptr(W2), _ptr(out), N, dm, dff, int(topk), _stream(stream))
    _check(rc, "topk_ffn_fwd_host")


# Size of the fixed scratch buffer of topk_ffn_fwd_noalloc (include/topk_attention.h).
TOPK_FFN_NOALLOC_SCRATCH_BYTES = 32 << 20


def topk_ffn_fwd_noalloc(x, W1, W2, out, topk: int, stream=None) -> None:
    """topk_ffn_fwd for callers that cannot allocate device memory at call time.

    Scratch comes from one fixed buffer inside the library instead of the
    stream-ordered pool (see the C header for the size limit and why calls
    that overlap on the GPU must be serialised).
    """
    N, dm, dff = _ffn_dims(x, W1, W2, out)
    rc = lib().topk_ffn_fwd_noalloc(_ptr(x), _ptr(W1), _ptr(W2), _ptr(out), N, dm, dff, int(topk), _stream(stream))
    _check(rc, "topk_ffn_fwd_noalloc")


def _cache_check(idx, score, rows_shape, topk):
    want = (*rows_shape, topk)
    for name, t, dt in (("idx", idx, torch.int32), ("score", score, torch.float32)):
        if t.dtype != dt or tuple(t.shape) != want or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous {list(want)} {dt} tensor")


def topk_attn_bwd(q, k, v, dout, idx, score, dq, dk, dv, stream=None) -> None:
    """Backward pass of Eq. 4 for the cached kept set (Sec. 2.2): fp32 dq [B,H,Lq,d], dk/dv [B,H,Lk,d]."""
    B, H, Lq, Lk, d = _attn_dims(q, k, v, dout)
    topk = idx.shape[-1]
    _cache_check(idx, score, (B, H, Lq), topk)
    for name, t, shape in (("dq", dq, (B, H, Lq, d)), ("dk", dk, (B, H, Lk, d)), ("dv", dv, (B, H, Lk, d))):
        if t.dtype != torch.float32 or tuple(t.shape) != shape or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous {list(shape)} float32 tensor")
    rc = lib().topk_attn_bwd(_ptr(q), _ptr(k), _ptr(v), _ptr(dout), _ptr(idx), _ptr(score), _ptr(dq), _ptr(dk),
                             _ptr(dv), B, H, Lq, Lk, d, int(topk), _dtype_code(q), _stream(stream))
    _check(rc, "topk_attn_bwd")


def topk_ffn_bwd(x, W1, W2, dout, idx, score, dx, dW1, dW2, stream=None) -> None:
    """Backward pass of the top-k FF layer (Eq. 3) for the cached kept set: fp32 dx, dW1, dW2."""
    N, dm, dff = _ffn_dims(x, W1, W2, dout)
    topk = idx.shape[-1]
    _cache_check(idx, score, (N,), topk)
    for name, t, shape in (("dx", dx, (N, dm)), ("dW1", dW1, (dff, dm)), ("dW2", dW2, (dff, dm))):
        if t.dtype != torch.float32 or tuple(t.shape) != shape or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous {list(shape)} float32 tensor")
    rc = lib().topk_ffn_bwd(_ptr(x), _ptr(W1), _ptr(W2), _ptr(dout), _ptr(idx), _ptr(score), _ptr(dx), _ptr(dW1),
                            _ptr(dW2), N, dm, dff, int(topk), _stream(stream))
    _check(rc, "topk_ffn_bwd")


def topk_attn_bwd_workspace_bytes(B, H, Lq, Lk, d, topk, dtype) -> int:
    return int(lib().topk_attn_bwd_workspace_bytes(B, H, Lq, Lk, d, topk, dtype))


def topk_ffn_bwd_workspace_bytes(N, d_model, d_ff, topk) -> int:
    return int(lib().topk_ffn_bwd_workspace_bytes(N, d_model, d_ff, topk))


def topk_attn_workspace_bytes(B, H, Lq, Lk, d, topk, chunk, dtype) -> int:
    return int(lib().topk_attn_workspace_bytes(B, H, Lq, Lk, d, topk, chunk, dtype))


def topk_ffn_workspace_bytes(N, d_model, d_ff, topk) -> int:
    return int(lib().topk_ffn_workspace_bytes(N, d_model, d_ff, topk))


def topk_check(stream=None) -> None:
    """Synchronise and raise if a kernel recorded a device-side error since the last check."""
    _check(lib().topk_check(_stream(stream)), "topk_check")


def topk_last_launch_count() -> int:
    return int(lib().topk_last_launch_count())


def topk_set_wait_limit_us(us: int) -> int:
    return int(lib().topk_set_wait_limit_us(int(us)))


def topk_pool_usage(reset_high: bool = False) -> tuple[int, int]:
    """(bytes in use at most since the last reset, bytes reserved now) of the library's own
    device-memory pool on the current device."""
    hi, res = ctypes.c_size_t(0), ctypes.c_size_t(0)
    _check(lib().topk_pool_usage(ctypes.byref(hi), ctypes.byref(res), int(bool(reset_high))), "topk_pool_usage")
    return int(hi.value), int(res.value)


def topk_pool_trim() -> None:
    """Hand the pool's reserved but unused device memory back (synchronise the streams first)."""
    _check(lib().topk_pool_trim(), "topk_pool_trim")


# convenience wrappers that allocate the outputs ---------------------------------------------

def attention(q, k, v, topk: int, chunk: int = 1024, causal: bool = False, return_indices: bool = False,
              stream=None, kv_len=None, mask=None):
    """Top-k attention; kv_len ([B] int32) and mask (bool [B|1, H|1, Lq, Lk], True = valid) add Eq. 2's
    general masks."""
    out = torch.empty_like(q)
    if kv_len is not None or mask is not None:
        B, H, Lq, _ = q.shape
        idx = score = None
        if return_indices:
            idx = torch.empty(B, H, Lq, topk, dtype=torch.int32, device=q.device)
            score = torch.empty(B, H, Lq, topk, dtype=torch.float32, device=q.device)
        words, bs, hs = pack_mask(mask) if mask is not None else (None, 0, 0)
        topk_attn_fwd_masked(q, k, v, out, topk, chunk, causal, kv_len, words, bs, hs, idx, score, stream)
        return (out, idx, score) if return_indices else out
    if not return_indices:
        topk_attn_fwd(q, k, v, out, topk, chunk, causal, stream)
        return out
    B, H, Lq, _ = q.shape
    idx = torch.empty(B, H, Lq, topk, dtype=torch.int32, device=q.device)
    score = torch.empty(B, H, Lq, topk, dtype=torch.float32, device=q.device)
    topk_attn_fwd_indices(q, k, v, out, topk, chunk, causal, idx, score, stream)
    return out, idx, score


def ffn(x, W1, W2, topk: int, return_indices: bool = False, stream=None):
    out = torch.empty(x.shape[0], x.shape[1], dtype=torch.float32, device=x.device)
    if not return_indices:
        topk_ffn_fwd(x, W1, W2, out, topk, stream)
        return out
    idx = torch.empty(x.shape[0], topk, dtype=torch.int32, device=x.device)
    score = torch.empty(x.shape[0], topk, dtype=torch.float32, device=x.device)
    topk_ffn_fwd_indices(x, W1, W2, out, topk, idx, score, stream)
    return out, idx, score


def attention_bwd(q, k, v, dout, idx, score, stream=None):
    """Gradients (dq, dk, dv), fp32, of top-k attention for the cache (idx, score) of attention(...,
    return_indices=True)."""
    dq = torch.empty(q.shape, dtype=torch.float32, device=q.device)
    dk = torch.empty(k.shape, dtype=torch.float32, device=k.device)
    dv = torch.empty(v.shape, dtype=torch.float32, device=v.device)
    topk_attn_bwd(q, k, v, dout, idx, score, dq, dk, dv, stream)
    return dq, dk, dv


def ffn_bwd(x, W1, W2, dout, idx, score, stream=None):
    """Gradients (dx, dW1, dW2), fp32, of the top-k FF layer for the cache of ffn(..., return_indices=True)."""
    dx = torch.empty(x.shape, dtype=torch.float32, device=x.device)
    dW1 = torch.empty(W1.shape, dtype=torch.float32, device=W1.device)
    dW2 = torch.empty(W2.shape, dtype=torch.float32, device=W2.device)
    topk_ffn_bwd(x, W1, W2, dout, idx, score, dx, dW1, dW2, stream)
    return dx, dW1, dW2
