"""Parity rules between the CUDA path and the CPU oracle -- TEST INFRASTRUCTURE ONLY.

Used by the GPU tests and by the benchmark's oracle leg (which checks the
timed call's output on the rows it times the oracle on).  The product path
never imports it.

For every checked row:

1. Index sets: the GPU's kept set must equal the oracle's, as a set, unless the
   row is a near tie: |s_(k) - s_(k+1)| < 1e-3 * max(|s_(k)|, |s_(k+1)|, 1e-3)
   (oracle scores; the floor keeps near-zero scores on an absolute 1e-6).
2. Validity on every row, near tie or not: each GPU-kept key, scored exactly by
   the oracle, must be at least the oracle's k-th score minus delta, where
   delta = d * 2^-22 * |q_i| * max_j |k_j| bounds the fp32 accumulation error
   of one score (products of bf16 values are exact in fp32).
3. Output: the GPU row must match the oracle's index-evaluate of the GPU's own
   kept set within `tol` (max abs); on rows with an exact set match that is
   the oracle's output itself.
4. The GPU's kept list is ordered by its own scores, non-increasing.
"""
from __future__ import annotations

import numpy as np
import torch

from . import SOFTMAX, eval_indices, topk_attention

TOL = {"bf16": 2e-2, "f32": 1e-5}


def near_tie(sk, sk1):
    with np.errstate(invalid="ignore"):  # rows with fewer than k + 1 valid keys compare -inf with -inf
        return np.abs(sk - sk1) < 1e-3 * np.maximum(np.maximum(np.abs(sk), np.abs(sk1)), 1e-3)


def _delta(q_rows: np.ndarray, k_all: torch.Tensor, d: int) -> np.ndarray:
    qn = np.linalg.norm(q_rows.astype(np.float64), axis=1)
    kn = float(torch.linalg.vector_norm(k_all.detach().float(), dim=-1).max())
    return d * 2.0 ** -22 * qn * kn + 1e-30


def check_rows(*, q, k, v, rows, gpu_out, gpu_idx, gpu_score, topk, dtype, act=SOFTMAX, causal=False,
               tol=None, ref=None, kv_len=None, mask=None):
    """q/k/v: CPU tensors [B,H,L,d]; rows: flattened row ids; gpu_*: CPU arrays for those rows;
    ref: the oracle's topk_attention result for those rows, if already computed; kv_len / mask: Eq. 2's
    masks as the oracle takes them.  Returns a dict of statistics; raises AssertionError on a violation."""
    tol = TOL[dtype] if tol is None else tol
    rows = np.asarray(rows, dtype=np.int64)
    if ref is None:
        ref = topk_attention(q, k, v, topk, act=act, causal=causal, rows=rows, kv_len=kv_len, mask=mask)
    gi = np.asarray(gpu_idx, dtype=np.int32).reshape(len(rows), topk)
    gs = np.asarray(gpu_score, dtype=np.float64).reshape(len(rows), topk)
    go = np.asarray(gpu_out, dtype=np.float64).reshape(len(rows), -1)
    B, H, Lq, d = q.shape
    Lk = k.shape[2]

    # kept counts and padding
    kept_ref = (ref["idx"] >= 0).sum(1)
    kept_gpu = (gi >= 0).sum(1)
    assert np.array_equal(kept_ref, kept_gpu), "kept counts differ"
    for r in range(len(rows)):
        n = kept_gpu[r]
        assert np.all(gi[r, n:] == -1) and np.all(gi[r, :n] >= 0) and np.all(gi[r, :n] < Lk)
        assert len(set(gi[r, :n].tolist())) == n, "duplicate index"
    if causal:
        i = (rows % Lq)[:, None]
        assert np.all((gi == -1) | (gi <= i + Lk - Lq)), "causal mask violated"
    if kv_len is not None:
        n_b = np.asarray(kv_len, dtype=np.int64)[rows // (H * Lq)][:, None]
        assert np.all((gi == -1) | (gi < n_b)), "key count violated"
    if mask is not None:
        m = np.asarray(mask, dtype=bool)
        for r in range(len(rows)):
            b, h, i_r = rows[r] // (H * Lq), (rows[r] // Lq) % H, rows[r] % Lq
            mr = m[b if m.shape[0] > 1 else 0, h if m.shape[1] > 1 else 0, i_r]
            picks = gi[r][gi[r] >= 0]
            assert np.all(mr[picks]), "bit mask violated"

    # order of the GPU list: its own scores non-increasing, equal scores by ascending index
    for r in range(len(rows)):
        n = kept_gpu[r]
        dsc = np.diff(gs[r, :n])
        assert np.all(dsc <= 0), "GPU list not ordered by score"
        eq = np.nonzero(dsc == 0)[0]
        assert np.all(gi[r, eq] < gi[r, eq + 1]), "equal scores not ordered by index"

    # exact oracle scores of the GPU's picks
    ev_out, ev_score = eval_indices(q, k, v, gi, act=act, rows=rows)
    kth = np.array([ref["score"][r, kept_ref[r] - 1] if kept_ref[r] > 0 else np.inf for r in range(len(rows))])
    qrows = _raw_rows(q, rows)
    delta = _delta(qrows, k, d)
    worst_pick = np.array([ev_score[r, :kept_gpu[r]].min() if kept_gpu[r] else np.inf for r in range(len(rows))])
    bad = worst_pick < kth - delta
    assert not bad.any(), f"{bad.sum()} rows keep a key scoring below the k-th oracle score minus delta"

    tie = near_tie(kth, ref["next_score"])
    same = np.array([set(gi[r].tolist()) == set(ref["idx"][r].tolist()) for r in range(len(rows))])
    mismatch = ~same & ~tie
    assert not mismatch.any(), f"{mismatch.sum()} rows with a clear gap select a different set"

    err_eval = np.abs(go - ev_out).max() if len(rows) else 0.0
    assert err_eval <= tol, f"output differs from index-evaluate by {err_eval} > {tol}"
    err_ref = np.abs(go[same] - ref["out"][same]).max() if same.any() else 0.0
    assert err_ref <= tol, f"output differs from oracle by {err_ref} > {tol}"
    return {"rows": len(rows), "near_tie_frac": float(tie.mean()), "exact_set_frac": float(same.mean()),
            "max_err": float(max(err_eval, err_ref))}


def _raw_rows(t, rows):
    a = t.detach().float().cpu().reshape(-1, t.shape[-1]).numpy()
    return a[rows]


def to_np(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy() if t.dtype == torch.bfloat16 else t.detach().cpu().numpy()
