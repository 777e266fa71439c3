"""Pins for the CPU oracle against things other than itself (CPU only).

Each check is fixed by the paper or by mathematics, not by re-typing the
oracle's own formula:

* Eq. 4 with k = L_K is Eq. 1: compared with torch's scaled_dot_product_attention
  (a library routine, fp64, scale 1 because lambda is folded into Q).
* Eq. 4 with the causal mask and k = L_K is Eq. 2 with the causal mask: SDPA is_causal.
* Eq. 3 with k = d_ff is the dense feed-forward layer ReLU(x W1^T) W2 (torch fp64).
* Selection against brute force: a full sort of every row on tiny inputs whose
  scores are exact dyadic numbers (so ties are frequent and exact), all k.
* Closed forms: identical keys keep keys 0..k-1 and average their values; causal
  row 0 returns v_0; causal rows i < k keep exactly {0..i}; k = 1 returns the
  value of the arg-max key; all-negative FF scores give 0; constant values give
  that constant; the output is linear in V.
* Invariant: permuting the keys with their values (Sec. 2.1: FF keys have no
  order) leaves the output unchanged and permutes the kept indices.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2106_06899_gb300 import workloads


def _f64(t):
    return t.to(torch.float64)


def _sdpa(q, k, v, causal=False):
    return torch.nn.functional.scaled_dot_product_attention(_f64(q), _f64(k), _f64(v), scale=1.0,
                                                            is_causal=causal)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_all_keys_equals_plain_attention(dtype):
    q, k, v = workloads.attention_inputs(2, 3, 37, 50, 16, dtype=dtype, seed=11)
    r = oracle.topk_attention(q, k, v, 50)
    ref = _sdpa(q, k, v).reshape(-1, 16).numpy()
    np.testing.assert_allclose(r["out"], ref, rtol=0, atol=1e-12)
    van = oracle.vanilla(q, k, v)
    np.testing.assert_allclose(van, ref, rtol=0, atol=1e-12)
    assert np.all(np.sort(r["idx"], axis=1) == np.arange(50)[None])
    assert np.all(np.isneginf(r["next_score"]))


def test_all_keys_causal_equals_masked_attention():
    q, k, v = workloads.attention_inputs(1, 2, 45, 45, 8, dtype="f32", seed=12)
    r = oracle.topk_attention(q, k, v, 45, causal=True)
    ref = _sdpa(q, k, v, causal=True).reshape(-1, 8).numpy()
    np.testing.assert_allclose(r["out"], ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(oracle.vanilla(q, k, v, causal=True), ref, rtol=0, atol=1e-12)


def test_ffn_all_keys_equals_dense_ffn():
    x, w1, w2 = workloads.ffn_inputs(19, 24, 40, dtype="bf16", seed=13)
    r = oracle.ffn(x, w1, w2, 40)
    ref = torch.relu(_f64(x) @ _f64(w1).T) @ _f64(w2)
    np.testing.assert_allclose(r["out"], ref.numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(oracle.ffn_dense(x, w1, w2), ref.numpy(), rtol=0, atol=1e-12)


def _dyadic(shape, rng):
    # multiples of 1/4 in [-1, 1]: every product and sum below is exact in fp32 and fp64
    return (rng.integers(-4, 5, size=shape) / 4.0).astype(np.float32)


def _bruteforce(q, k, v, topk, causal, act):
    """Full sort of every row by (score desc, index asc); scores by numpy matmul in fp64."""
    B, H, Lq, d = q.shape
    Lk = k.shape[2]
    s = np.einsum("bhid,bhjd->bhij", q.astype(np.float64), k.astype(np.float64)).reshape(B * H, Lq, Lk)
    vv = v.astype(np.float64).reshape(B * H, Lk, d)
    outs, idxs, nexts = [], [], []
    for bh in range(B * H):
        for i in range(Lq):
            n = min(i + 1, Lk) if causal else Lk
            row = s[bh, i, :n]
            order = np.lexsort((np.arange(n), -row))  # primary: -score, secondary: index
            keep = order[:topk]
            sk = row[keep]
            if act == oracle.SOFTMAX:
                w = np.exp(sk - sk.max())
                w /= w.sum()
            else:
                w = np.maximum(sk, 0.0)
            outs.append(w @ vv[bh, keep])
            idxs.append(np.concatenate([keep, -np.ones(topk - len(keep), np.int64)]))
            nexts.append(row[order[topk]] if n > topk else -np.inf)
    return np.array(outs), np.array(idxs), np.array(nexts)


@pytest.mark.parametrize("causal", [False, True])
@pytest.mark.parametrize("act", [oracle.SOFTMAX, oracle.RELU])
def test_selection_matches_full_sort(causal, act):
    rng = np.random.default_rng(5)
    B, H, L, d = 1, 2, 24, 3
    q, k, v = _dyadic((B, H, L, d), rng), _dyadic((B, H, L, d), rng), _dyadic((B, H, L, d), rng)
    for topk in range(1, L + 1):
        r = oracle.topk_attention(q, k, v, topk, act=act, causal=causal)
        out, idx, nxt = _bruteforce(q, k, v, topk, causal, act)
        assert np.array_equal(r["idx"], idx), topk
        np.testing.assert_allclose(r["out"], out, rtol=0, atol=1e-12)
        np.testing.assert_array_equal(r["next_score"], nxt)


def test_ties_go_to_lower_index():
    # identical keys: every score of a row ties, so the first k keys are kept
    L, d, topk = 40, 4, 7
    rng = np.random.default_rng(3)
    q = rng.standard_normal((1, 1, 5, d)).astype(np.float32)
    k = np.tile(rng.standard_normal((1, 1, 1, d)).astype(np.float32), (1, 1, L, 1))
    v = rng.standard_normal((1, 1, L, d)).astype(np.float32)
    r = oracle.topk_attention(q, k, v, topk)
    assert np.all(r["idx"] == np.arange(topk)[None])
    np.testing.assert_allclose(r["out"], np.tile(v[0, 0, :topk].astype(np.float64).mean(0), (5, 1)), atol=1e-12)


def test_ties_structured():
    # keys cycle through 3 exact score levels 2 > 1 > 0; top-k takes the level-2 keys
    # in index order, then the level-1 keys in index order
    L, topk = 30, 14
    q = np.array([[[[1.0, 0.0]]]], np.float32)
    k = np.zeros((1, 1, L, 2), np.float32)
    k[0, 0, :, 0] = np.array([j % 3 for j in range(L)], np.float32)  # score of key j = j mod 3
    v = np.zeros((1, 1, L, 2), np.float32)
    r = oracle.topk_attention(q, k, v, topk)
    twos = [j for j in range(L) if j % 3 == 2]
    ones = [j for j in range(L) if j % 3 == 1]
    assert list(r["idx"][0]) == (twos + ones)[:topk]
    assert r["next_score"][0] == 1.0  # the 15th entry is the next level-1 key


def test_causal_closed_forms():
    q, k, v = workloads.attention_inputs(1, 1, 64, 64, 16, dtype="f32", seed=4)
    topk = 10
    r = oracle.topk_attention(q, k, v, topk, causal=True)
    i = np.arange(64)[:, None]
    idx = r["idx"]
    assert np.all((idx == -1) | (idx <= i))  # no future key is ever kept
    for row in range(topk):
        assert sorted(idx[row][idx[row] >= 0].tolist()) == list(range(row + 1))
        assert np.all(idx[row][row + 1:] == -1)
    np.testing.assert_array_equal(r["out"][0], v[0, 0, 0].double().numpy())  # softmax of one entry is 1
    assert np.all(idx[topk:] >= 0)


def test_k1_is_argmax_value():
    q, k, v = workloads.attention_inputs(2, 2, 9, 33, 8, dtype="f32", seed=8)
    r = oracle.topk_attention(q, k, v, 1)
    s = np.einsum("bhid,bhjd->bhij", q.double().numpy(), k.double().numpy())
    am = s.argmax(-1).reshape(-1)
    assert np.array_equal(r["idx"][:, 0], am)
    vv = v.double().numpy().reshape(4, 33, 8)
    np.testing.assert_array_equal(r["out"], vv[np.repeat(np.arange(4), 9), am])


def test_relu_drops_negative_selected_scores():
    x = np.ones((3, 4), np.float32)
    w1 = -np.abs(np.random.default_rng(1).standard_normal((12, 4))).astype(np.float32) - 0.1
    w2 = np.random.default_rng(2).standard_normal((12, 4)).astype(np.float32)
    r = oracle.ffn(x, w1, w2, 5)
    assert np.all(r["score"] < 0)
    np.testing.assert_array_equal(r["out"], 0.0)


def test_ffn_worked_example():
    # x = (1, 2); key rows give scores (1, 2, 3, -1, 0); top-2 keeps keys 2 and 1 (Eq. 3, Eq. 4)
    x = np.array([[1.0, 2.0]], np.float32)
    w1 = np.array([[1, 0], [0, 1], [1, 1], [-1, 0], [0, 0]], np.float32)
    w2 = np.array([[1, 1], [10, 0], [0, 100], [5, 5], [7, 7]], np.float32)
    r = oracle.ffn(x, w1, w2, 2)
    assert list(r["idx"][0]) == [2, 1]
    assert list(r["score"][0]) == [3.0, 2.0]
    assert list(r["out"][0]) == [20.0, 300.0]  # 3 * (0, 100) + 2 * (10, 0)
    assert r["next_score"][0] == 1.0


def test_softmax_weights_sum_to_one_and_linear_in_v():
    q, k, v = workloads.attention_inputs(1, 2, 20, 70, 8, dtype="f32", seed=21)
    ones = torch.full_like(v, 0.75)
    r = oracle.topk_attention(q, k, ones, 9)
    np.testing.assert_allclose(r["out"], 0.75, rtol=0, atol=1e-14)
    v2 = torch.randn(v.shape, generator=torch.Generator().manual_seed(3))
    a = oracle.topk_attention(q, k, v, 9)["out"]
    b = oracle.topk_attention(q, k, v2, 9)["out"]
    c = oracle.topk_attention(q, k, (v.double() + v2.double()).float(), 9)["out"]
    # v + v2 is rounded to fp32 before the oracle sees it; compare against the same rounding
    np.testing.assert_allclose(c, a + b, rtol=0, atol=1e-6)


@pytest.mark.parametrize("act", [oracle.SOFTMAX, oracle.RELU])
def test_key_permutation_equivariance(act):
    q, k, v = workloads.attention_inputs(1, 1, 16, 90, 8, dtype="f32", seed=31)
    perm = torch.randperm(90, generator=torch.Generator().manual_seed(1))
    a = oracle.topk_attention(q, k, v, 12, act=act)
    b = oracle.topk_attention(q, k[:, :, perm], v[:, :, perm], 12, act=act)
    np.testing.assert_allclose(a["out"], b["out"], rtol=0, atol=1e-12)
    assert np.array_equal(perm.numpy()[b["idx"]], a["idx"])


def test_eval_indices_reproduces_selection():
    q, k, v = workloads.attention_inputs(2, 2, 30, 64, 16, dtype="bf16", seed=41)
    rows = np.array([0, 5, 31, 77, 119])
    r = oracle.topk_attention(q, k, v, 8, rows=rows)
    out, score = oracle.eval_indices(q, k, v, r["idx"], rows=rows)
    np.testing.assert_array_equal(out, r["out"])
    np.testing.assert_array_equal(score, r["score"])
    # a row subset gives the same numbers as the full run
    full = oracle.topk_attention(q, k, v, 8)
    np.testing.assert_array_equal(full["out"][rows], r["out"])


def test_bf16_widening_is_exact():
    # bf16 values are read exactly: 1 + 2^-7 survives, a dot product of them is exact
    t = torch.tensor([[[[1.0 + 2 ** -7, -3.0]]]], dtype=torch.bfloat16)
    kk = torch.tensor([[[[2.0, 0.5]]]], dtype=torch.bfloat16)
    vv = torch.tensor([[[[1.0, 2.0]]]], dtype=torch.bfloat16)
    r = oracle.topk_attention(t, kk, vv, 1)
    assert r["score"][0, 0] == (1.0 + 2 ** -7) * 2.0 - 1.5
