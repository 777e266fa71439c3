"""CPU oracle for top-k attention -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The
product path (``paper_2106_06899_gb300``) never imports, links or runs it.

It wraps ``topk_oracle.c`` (plain C, fp64, one pthread per host core), which
computes the paper's definitions directly:

* Eq. 4 -- top-k attention: keep the k largest scores of each row of Q K^T,
  softmax over those k only, weighted sum of the matching value rows;
* Eq. 3 -- the feed-forward layer cast as attention: Q = x, K = W1, V = W2,
  ReLU in place of softmax;
* Eq. 1 / Eq. 2 -- plain (optionally causal) attention over every key, the
  special case top-k reduces to when k equals the number of keys;
* index-evaluate mode: the same activation and weighted sum for a given
  kept set (used where the near-tie rule lets two correct sets differ);
* the backward pass for a given kept set (Sec. 2.2): gradients with respect
  to Q, K, V (x, W1, W2 for the feed-forward layer), the kept set being the
  forward pass's cache.

Ties are broken toward the lower key index; causal rows with fewer than k
valid keys keep all of them.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "topk_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

F32, BF16, F64 = 0, 1, 2
SOFTMAX, RELU = 0, 1


def build(force: bool = False) -> str:
    """Compile topk_oracle.c into liboracle.so (gcc -O2, no fast-math)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.run(
            ["gcc", "-O2", "-std=c11", "-D_POSIX_C_SOURCE=200809L", "-shared", "-fPIC", "-pthread",
             "-o", tmp, _SRC, "-lm"],
            check=True,
        )
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            i64, i32, vp = ctypes.c_int64, ctypes.c_int, ctypes.c_void_p
            lib.oracle_topk.argtypes = [i32, i32, vp, vp, vp, i64, i64, i64, i64, i64, i64, i32, vp, i64,
                                        vp, vp, vp, vp, i32]
            lib.oracle_vanilla.argtypes = [i32, i32, vp, vp, vp, i64, i64, i64, i64, i64, i32, vp, i64, vp, i32]
            lib.oracle_eval_indices.argtypes = [i32, i32, vp, vp, vp, i64, i64, i64, i64, i64, i64, vp, i64,
                                                vp, vp, vp, vp, i32]
            lib.oracle_topk_masked.argtypes = [i32, i32, vp, vp, vp, i64, i64, i64, i64, i64, i64, i32, vp, vp,
                                               i64, i64, vp, i64, vp, vp, vp, vp, i32]
            lib.oracle_vanilla_masked.argtypes = [i32, i32, vp, vp, vp, i64, i64, i64, i64, i64, i32, vp, vp,
                                                  i64, i64, vp, i64, vp, i32]
            lib.oracle_topk_bwd.argtypes = [i32, i32, vp, vp, vp, i32, vp, i64, i64, i64, i64, i64, i64, vp,
                                            vp, vp, vp, i32]
            lib.oracle_hardware_threads.argtypes = []
            for f in (lib.oracle_topk, lib.oracle_vanilla, lib.oracle_eval_indices, lib.oracle_topk_bwd,
                      lib.oracle_topk_masked, lib.oracle_vanilla_masked, lib.oracle_hardware_threads):
                f.restype = ctypes.c_int
            _lib = lib
    return _lib


def hardware_threads() -> int:
    return int(_load().oracle_hardware_threads())


def _as_raw(a):
    """numpy float32 / float64 / uint16(bf16 bits) array, or a CPU torch tensor -> (contiguous ndarray, dtype code)."""
    if not isinstance(a, np.ndarray):  # torch tensor
        import torch

        t = a.detach().cpu().contiguous()
        if t.dtype == torch.bfloat16:
            return t.view(torch.int16).numpy().view(np.uint16), BF16
        if t.dtype == torch.float32:
            return t.numpy(), F32
        if t.dtype == torch.float64:
            return t.numpy(), F64
        raise TypeError(f"oracle takes float32, float64 or bfloat16, got {t.dtype}")
    a = np.ascontiguousarray(a)
    if a.dtype == np.float32:
        return a, F32
    if a.dtype == np.float64:
        return a, F64
    if a.dtype == np.uint16:
        return a, BF16
    raise TypeError(f"oracle takes float32, float64 or bf16-as-uint16 arrays, got {a.dtype}")


def _rows_arg(rows, total):
    if rows is None:
        return None, total, None
    r = np.ascontiguousarray(np.asarray(rows, dtype=np.int64))
    if r.size and (r.min() < 0 or r.max() >= total):
        raise ValueError("row index out of range")
    return r, r.size, r.ctypes.data


def _common(q, k, v, act):
    qa, dt = _as_raw(q)
    ka, dt2 = _as_raw(k)
    va, dt3 = _as_raw(v)
    if not (dt == dt2 == dt3):
        raise TypeError("q, k, v must share a dtype")
    return qa, ka, va, dt


def _masks(kv_len, mask, B, H, Lq, Lk):
    """(kv_len int32 [B] or None, packed mask words or None, batch stride, head stride).

    mask: boolean array of shape [B or 1, H or 1, Lq, Lk], True where the key is valid (Eq. 2's
    B_ij = 0); a dimension of size 1 applies to every batch / head.  Packed here, independently of
    the CUDA binding, as bit j % 32 of word j // 32 of each query row (little-endian bit order)."""
    kl = None
    if kv_len is not None:
        kl = np.ascontiguousarray(np.asarray(kv_len, dtype=np.int32).reshape(B))
    words = None
    mbs = mhs = 0
    if mask is not None:
        m = np.asarray(mask, dtype=bool)
        if m.ndim != 4 or m.shape[2:] != (Lq, Lk) or m.shape[0] not in (1, B) or m.shape[1] not in (1, H):
            raise ValueError("mask must be [B or 1, H or 1, Lq, Lk]")
        W = (Lk + 31) // 32
        padded = np.zeros(m.shape[:3] + (W * 32,), bool)
        padded[..., :Lk] = m
        bits = padded.reshape(m.shape[:3] + (W, 32)).astype(np.uint64)
        words = np.ascontiguousarray((bits << np.arange(32, dtype=np.uint64)).sum(axis=-1).astype(np.uint32))
        mhs = Lq * W if m.shape[1] == H and H > 1 else 0
        mbs = m.shape[1] * Lq * W if m.shape[0] == B and B > 1 else 0
    return kl, words, mbs, mhs


def _ptr(a):
    return None if a is None else a.ctypes.data


def topk_attention(q, k, v, topk: int, *, act: int = SOFTMAX, causal: bool = False, rows=None, threads: int = 0,
                   kv_len=None, mask=None):
    """Eq. 4 (act=SOFTMAX) or Eq. 3 (act=RELU) for q [B,H,Lq,d], k/v [B,H,Lk,d], under the masks of
    Eq. 2: causal (key j valid for query i iff j <= i + Lk - Lq; needs Lq <= Lk), kv_len ([B]: key j
    valid iff j < kv_len[b]) and mask (boolean [B|1, H|1, Lq, Lk], True = valid).

    Returns dict(out [n,d] f64, idx [n,topk] i32 (-1 pad), score [n,topk] f64 (-inf pad),
    next_score [n] f64 (the (k+1)-th score, -inf if none)); n = len(rows) or B*H*Lq.
    """
    qa, ka, va, dt = _common(q, k, v, act)
    B, H, Lq, d = qa.shape
    Lk = ka.shape[2]
    if ka.shape != (B, H, Lk, d) or va.shape != (B, H, Lk, d):
        raise ValueError("shape mismatch")
    r, n, rp = _rows_arg(rows, B * H * Lq)
    kl, words, mbs, mhs = _masks(kv_len, mask, B, H, Lq, Lk)
    out = np.zeros((n, d), np.float64)
    idx = np.zeros((n, topk), np.int32)
    score = np.zeros((n, topk), np.float64)
    nxt = np.zeros((n,), np.float64)
    rc = _load().oracle_topk_masked(act, dt, qa.ctypes.data, ka.ctypes.data, va.ctypes.data, B, H, Lq, Lk, d,
                                    topk, int(causal), _ptr(kl), _ptr(words), mbs, mhs, rp, n, out.ctypes.data,
                                    idx.ctypes.data, score.ctypes.data, nxt.ctypes.data, threads)
    if rc:
        raise RuntimeError(f"oracle_topk failed: {rc}")
    return {"out": out, "idx": idx, "score": score, "next_score": nxt}


def vanilla(q, k, v, *, act: int = SOFTMAX, causal: bool = False, rows=None, threads: int = 0, kv_len=None,
            mask=None):
    """Eq. 1 (softmax over all valid keys under the masks of Eq. 2, as in topk_attention) -> out [n, d] f64."""
    qa, ka, va, dt = _common(q, k, v, act)
    B, H, Lq, d = qa.shape
    Lk = ka.shape[2]
    r, n, rp = _rows_arg(rows, B * H * Lq)
    kl, words, mbs, mhs = _masks(kv_len, mask, B, H, Lq, Lk)
    out = np.zeros((n, d), np.float64)
    rc = _load().oracle_vanilla_masked(act, dt, qa.ctypes.data, ka.ctypes.data, va.ctypes.data, B, H, Lq, Lk, d,
                                       int(causal), _ptr(kl), _ptr(words), mbs, mhs, rp, n, out.ctypes.data,
                                       threads)
    if rc:
        raise RuntimeError(f"oracle_vanilla failed: {rc}")
    return out


def eval_indices(q, k, v, idx, *, act: int = SOFTMAX, rows=None, threads: int = 0, return_idx: bool = False):
    """Index-evaluate: given kept sets idx [n, topk] (-1 = empty), return (out [n,d], score [n,topk]).

    score lists each row's kept entries in the total order (score descending, index
    ascending), -inf padded; with return_idx the matching indices (-1 padded) come third."""
    qa, ka, va, dt = _common(q, k, v, act)
    B, H, Lq, d = qa.shape
    Lk = ka.shape[2]
    r, n, rp = _rows_arg(rows, B * H * Lq)
    ia = np.ascontiguousarray(np.asarray(idx, dtype=np.int32))
    if ia.shape[0] != n:
        raise ValueError("idx rows must match the listed rows")
    K = ia.shape[1]
    out = np.zeros((n, d), np.float64)
    score = np.zeros((n, K), np.float64)
    iout = np.zeros((n, K), np.int32) if return_idx else None
    rc = _load().oracle_eval_indices(act, dt, qa.ctypes.data, ka.ctypes.data, va.ctypes.data, B, H, Lq, Lk, d,
                                     K, rp, n, ia.ctypes.data, out.ctypes.data, score.ctypes.data,
                                     None if iout is None else iout.ctypes.data, threads)
    if rc:
        raise RuntimeError(f"oracle_eval_indices failed: {rc}")
    return (out, score, iout) if return_idx else (out, score)


def ffn(x, W1, W2, topk: int, *, rows=None, threads: int = 0):
    """Eq. 3 with top-k: x [N, dm], W1/W2 [d_ff, dm] -> same dict as topk()."""
    return topk_attention(x[None, None], W1[None, None], W2[None, None], topk, act=RELU, rows=rows,
                             threads=threads)


def ffn_dense(x, W1, W2, *, rows=None, threads: int = 0):
    """Eq. 3 without top-k: ReLU(x W1^T) W2 over every key -> [n, dm] f64."""
    return vanilla(x[None, None], W1[None, None], W2[None, None], act=RELU, rows=rows, threads=threads)


def ffn_eval_indices(x, W1, W2, idx, *, rows=None, threads: int = 0):
    return eval_indices(x[None, None], W1[None, None], W2[None, None], idx, act=RELU, rows=rows,
                        threads=threads)


def topk_attention_bwd(q, k, v, dout, idx, *, act: int = SOFTMAX, threads: int = 0):
    """Backward pass of Eq. 4 (act=SOFTMAX) or Eq. 3 (act=RELU) for the kept sets idx.

    q [B,H,Lq,d], k/v [B,H,Lk,d], dout [B,H,Lq,d] (any dtype the oracle reads), idx [B*H*Lq, topk]
    int32 (-1 = empty slot).  Returns dict(dq [B,H,Lq,d], dk [B,H,Lk,d], dv [B,H,Lk,d]) in float64.
    """
    qa, ka, va, dt = _common(q, k, v, act)
    ga, gdt = _as_raw(dout)
    B, H, Lq, d = qa.shape
    Lk = ka.shape[2]
    if ka.shape != (B, H, Lk, d) or va.shape != (B, H, Lk, d) or ga.shape != (B, H, Lq, d):
        raise ValueError("shape mismatch")
    ia = np.ascontiguousarray(np.asarray(idx, dtype=np.int32))
    if ia.ndim != 2 or ia.shape[0] != B * H * Lq:
        raise ValueError("idx must be [B*H*Lq, topk]")
    dq = np.zeros((B, H, Lq, d), np.float64)
    dk = np.zeros((B, H, Lk, d), np.float64)
    dv = np.zeros((B, H, Lk, d), np.float64)
    rc = _load().oracle_topk_bwd(act, dt, qa.ctypes.data, ka.ctypes.data, va.ctypes.data, gdt, ga.ctypes.data,
                                 B, H, Lq, Lk, d, ia.shape[1], ia.ctypes.data, dq.ctypes.data, dk.ctypes.data,
                                 dv.ctypes.data, threads)
    if rc:
        raise RuntimeError(f"oracle_topk_bwd failed: {rc}")
    return {"dq": dq, "dk": dk, "dv": dv}


def ffn_bwd(x, W1, W2, dout, idx, *, threads: int = 0):
    """Backward pass of the top-k feed-forward layer (Eq. 3): x [N,dm], W1/W2 [d_ff,dm], dout [N,dm],
    idx [N, topk] -> dict(dx [N,dm], dW1 [d_ff,dm], dW2 [d_ff,dm]) in float64."""
    g = topk_attention_bwd(x[None, None], W1[None, None], W2[None, None], dout[None, None], idx, act=RELU,
                           threads=threads)
    return {"dx": g["dq"][0, 0], "dW1": g["dk"][0, 0], "dW2": g["dv"][0, 0]}
