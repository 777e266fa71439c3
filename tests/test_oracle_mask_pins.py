"""Pins for the oracle's masks (Eq. 2), CPU only.

A mask sets B_ij = -inf for the (query, key) pairs it excludes; top-k then
selects among the remaining keys.  Each check is fixed by something other
than the oracle's own mask code:

* an arbitrary boolean mask with k = L_K equals torch's scaled_dot_product_attention
  with the same boolean attn_mask (a library routine, fp64, scale 1);
* selection under a mask against brute force: a full sort of every row's valid
  keys on tiny inputs with exact dyadic scores (many ties), every k;
* per-batch key counts equal running each batch on its first kv_len[b] keys
  alone (closed form: the keys past the count are cut off);
* causal with Lq < Lk (queries are the last Lq positions) equals the last Lq
  rows of the causal problem with Lq = Lk; Lq = 1 equals attention over all keys;
* a row with no valid key outputs zeros and keeps nothing.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2106_06899_gb300 import workloads


def _f64(t):
    return t.to(torch.float64)


def _random_mask(shape, seed, p=0.6, ensure_row=True):
    rng = np.random.default_rng(seed)
    m = rng.random(shape) < p
    if ensure_row:  # at least one valid key per row (SDPA's softmax is undefined otherwise)
        m[..., 0] |= ~m.any(axis=-1)
    return m


@pytest.mark.parametrize("mshape", ["full", "per_batch", "shared"])
def test_mask_all_keys_equals_sdpa_with_mask(mshape):
    B, H, Lq, Lk, d = 2, 3, 29, 41, 16
    q, k, v = workloads.attention_inputs(B, H, Lq, Lk, d, dtype="bf16", seed=70)
    shape = {"full": (B, H, Lq, Lk), "per_batch": (B, 1, Lq, Lk), "shared": (1, 1, Lq, Lk)}[mshape]
    m = _random_mask(shape, 71)
    r = oracle.topk_attention(q, k, v, Lk, mask=m)
    ref = torch.nn.functional.scaled_dot_product_attention(_f64(q), _f64(k), _f64(v), scale=1.0,
                                                           attn_mask=torch.from_numpy(m))
    np.testing.assert_allclose(r["out"], ref.reshape(-1, d).numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(oracle.vanilla(q, k, v, mask=m), ref.reshape(-1, d).numpy(), rtol=0, atol=1e-12)
    kept = (r["idx"] >= 0).sum(axis=1)
    assert np.array_equal(kept, np.broadcast_to(m, (B, H, Lq, Lk)).reshape(-1, Lk).sum(axis=1))


@pytest.mark.parametrize("act", [oracle.SOFTMAX, oracle.RELU])
def test_masked_selection_matches_full_sort(act):
    B, H, Lq, Lk, d = 1, 2, 12, 40, 4
    rng = np.random.default_rng(72)
    # dyadic values: exact scores, frequent exact ties
    q = torch.from_numpy(rng.integers(-2, 3, (B, H, Lq, d)).astype(np.float32) / 2)
    k = torch.from_numpy(rng.integers(-2, 3, (B, H, Lk, d)).astype(np.float32) / 2)
    v = torch.from_numpy(rng.standard_normal((B, H, Lk, d)).astype(np.float32))
    m = _random_mask((B, H, Lq, Lk), 73, p=0.5, ensure_row=False)
    m[0, 0, 3] = False  # one row with no valid key
    s = (q.double() @ k.double().transpose(-1, -2)).numpy().reshape(-1, Lk)
    mm = m.reshape(-1, Lk)
    for topk in (1, 3, 7, 20, 40):
        r = oracle.topk_attention(q, k, v, topk, act=act, mask=m)
        for row in range(B * H * Lq):
            valid = np.nonzero(mm[row])[0]
            order = valid[np.lexsort((valid, -s[row, valid]))]  # score descending, index ascending
            want = order[:topk]
            got = r["idx"][row]
            assert np.array_equal(got[: len(want)], want), (topk, row)
            assert np.all(got[len(want):] == -1)
            nxt = s[row, order[topk]] if len(order) > topk else -np.inf
            assert r["next_score"][row] == nxt


def test_kv_len_equals_cut_keys():
    B, H, Lq, Lk, d, topk = 3, 2, 17, 50, 8, 6
    q, k, v = workloads.attention_inputs(B, H, Lq, Lk, d, dtype="f32", seed=74)
    kv_len = np.array([50, 23, 4], np.int32)  # the last batch has fewer keys than k
    r = oracle.topk_attention(q, k, v, topk, kv_len=kv_len)
    for b, n in enumerate(kv_len):
        cut = oracle.topk_attention(q[b:b + 1], k[b:b + 1, :, :n].contiguous(), v[b:b + 1, :, :n].contiguous(),
                                    min(topk, int(n)))
        rows = slice(b * H * Lq, (b + 1) * H * Lq)
        np.testing.assert_array_equal(r["out"][rows], cut["out"])
        kk = min(topk, int(n))
        np.testing.assert_array_equal(r["idx"][rows, :kk], cut["idx"])
        assert np.all(r["idx"][rows, kk:] == -1)


def test_kv_len_zero_outputs_zeros():
    B, H, L, d = 2, 1, 9, 8
    q, k, v = workloads.attention_inputs(B, H, L, L, d, dtype="f32", seed=75)
    r = oracle.topk_attention(q, k, v, 4, kv_len=np.array([0, 9], np.int32))
    first = slice(0, H * L)
    assert np.all(r["out"][first] == 0) and np.all(r["idx"][first] == -1)
    assert np.all(np.isneginf(r["score"][first])) and np.all(np.isneginf(r["next_score"][first]))
    assert np.all(r["idx"][H * L:] >= 0)


@pytest.mark.parametrize("act", [oracle.SOFTMAX, oracle.RELU])
def test_causal_decode_equals_last_rows_of_full_causal(act):
    B, H, Lk, d, topk = 1, 2, 60, 16, 8
    q, k, v = workloads.attention_inputs(B, H, Lk, Lk, d, dtype="bf16", seed=76)
    full = oracle.topk_attention(q, k, v, topk, act=act, causal=True)
    for Lq in (1, 5, 33):
        qd = q[:, :, Lk - Lq:].contiguous()
        dec = oracle.topk_attention(qd, k, v, topk, act=act, causal=True)
        want = np.concatenate([np.arange(h * Lk + Lk - Lq, (h + 1) * Lk) for h in range(H)])
        np.testing.assert_array_equal(dec["out"], full["out"][want])
        np.testing.assert_array_equal(dec["idx"], full["idx"][want])
    one = oracle.topk_attention(q[:, :, -1:].contiguous(), k, v, topk, act=act, causal=True)
    free = oracle.topk_attention(q[:, :, -1:].contiguous(), k, v, topk, act=act)
    np.testing.assert_array_equal(one["out"], free["out"])


def test_causal_requires_fewer_queries_than_keys():
    q, k, v = workloads.attention_inputs(1, 1, 10, 8, 8, dtype="f32", seed=77)
    with pytest.raises(RuntimeError):
        oracle.topk_attention(q, k, v, 4, causal=True)
