"""Pins for the oracle's backward pass (CPU only).

The backward pass of Sec. 2.2 differentiates Eq. 4 (Eq. 3) with the kept set
held fixed: the set is the forward pass's cache.  Nothing here re-types the
oracle's gradient formulas; each check is fixed by something else:

* autograd: torch's reverse mode, in fp64, through the forward definition
  written densely (the scores of keys outside the kept set masked to -inf
  before the softmax, or zeroed after the ReLU), for any kept set, causal
  rows with fewer than k keys included;
* the special case k = L_K: autograd through torch's scaled_dot_product_attention
  (plain attention, Eq. 1 / Eq. 2) and through the dense feed-forward layer;
* central finite differences of the oracle's own forward (index-evaluate
  mode, pinned separately against SDPA) on fp64 inputs;
* invariants: the softmax weights of a row sum to one, so its score
  gradients sum to zero (the rows of dK sum to zero over the keys) and the
  rows of dV sum to the rows of dout; keys never kept get no gradient.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2106_06899_gb300 import workloads


def _f64(t):
    return t.detach().to(torch.float64).clone().requires_grad_(True)


def _dense_mask(idx, B, H, Lq, Lk):
    """Boolean [B,H,Lq,Lk] of the kept pairs (idx [B*H*Lq, k], -1 = empty)."""
    m = np.zeros((B * H * Lq, Lk), bool)
    for r in range(idx.shape[0]):
        for j in idx[r]:
            if j >= 0:
                m[r, j] = True
    return torch.from_numpy(m.reshape(B, H, Lq, Lk))


def _autograd_masked(q, k, v, dout, mask, act):
    """Reverse mode of Eq. 4 / Eq. 3 written densely over the kept pairs (fp64)."""
    q64, k64, v64 = _f64(q), _f64(k), _f64(v)
    s = q64 @ k64.transpose(-1, -2)
    if act == oracle.SOFTMAX:
        w = torch.softmax(s.masked_fill(~mask, float("-inf")), dim=-1)
        w = torch.nan_to_num(w, nan=0.0)  # rows with no kept key
    else:
        w = torch.relu(s) * mask
    out = w @ v64
    (out * dout.to(torch.float64)).sum().backward()
    return q64.grad.numpy(), k64.grad.numpy(), v64.grad.numpy()


def _dout(shape, seed, dtype=torch.float32):
    g = torch.Generator().manual_seed(seed)
    return torch.randn(shape, generator=g).to(dtype)


def _random_sets(B, H, Lq, Lk, k, seed, causal=False, empty_frac=0.0):
    """Arbitrary kept sets (not the top k): distinct keys per row, some slots empty."""
    rng = np.random.default_rng(seed)
    idx = np.full((B * H * Lq, k), -1, np.int32)
    for r in range(B * H * Lq):
        i = r % Lq
        n_valid = min(i + 1, Lk) if causal else Lk
        take = min(k, n_valid)
        idx[r, :take] = rng.choice(n_valid, size=take, replace=False)
        drop = rng.random(k) < empty_frac
        idx[r, drop] = -1
        rng.shuffle(idx[r])
    return idx


@pytest.mark.parametrize("act", [oracle.SOFTMAX, oracle.RELU])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_bwd_matches_autograd_on_arbitrary_kept_sets(act, dtype):
    B, H, Lq, Lk, d, k = 2, 2, 23, 31, 8, 6
    q, kk, v = workloads.attention_inputs(B, H, Lq, Lk, d, dtype=dtype, seed=21)
    dout = _dout((B, H, Lq, d), 22)
    idx = _random_sets(B, H, Lq, Lk, k, seed=23, empty_frac=0.2)
    idx[5] = -1  # a row with no kept key has no gradient
    g = oracle.topk_attention_bwd(q, kk, v, dout, idx, act=act)
    rq, rk, rv = _autograd_masked(q, kk, v, dout, _dense_mask(idx, B, H, Lq, Lk), act)
    np.testing.assert_allclose(g["dq"], rq, rtol=0, atol=1e-12)
    np.testing.assert_allclose(g["dk"], rk, rtol=0, atol=1e-12)
    np.testing.assert_allclose(g["dv"], rv, rtol=0, atol=1e-12)
    assert np.all(g["dq"].reshape(-1, d)[5] == 0)


@pytest.mark.parametrize("act", [oracle.SOFTMAX, oracle.RELU])
def test_bwd_on_topk_sets_causal(act):
    """The forward pass's own kept sets, causal: rows i < k keep fewer than k keys (-1 padded)."""
    B, H, L, d, k = 1, 3, 40, 16, 8
    q, kk, v = workloads.attention_inputs(B, H, L, L, d, dtype="f32", seed=24)
    dout = _dout((B, H, L, d), 25)
    fwd = oracle.topk_attention(q, kk, v, k, act=act, causal=True)
    assert np.any(fwd["idx"] < 0)
    g = oracle.topk_attention_bwd(q, kk, v, dout, fwd["idx"], act=act)
    rq, rk, rv = _autograd_masked(q, kk, v, dout, _dense_mask(fwd["idx"], B, H, L, L), act)
    np.testing.assert_allclose(g["dq"], rq, rtol=0, atol=1e-12)
    np.testing.assert_allclose(g["dk"], rk, rtol=0, atol=1e-12)
    np.testing.assert_allclose(g["dv"], rv, rtol=0, atol=1e-12)


@pytest.mark.parametrize("causal", [False, True])
def test_bwd_all_keys_equals_sdpa_gradient(causal):
    """k = L_K keeps every valid key: the gradient of plain attention (SDPA, a library routine)."""
    B, H, L, d = 2, 2, 33, 16
    q, kk, v = workloads.attention_inputs(B, H, L, L, d, dtype="bf16", seed=26)
    dout = _dout((B, H, L, d), 27)
    fwd = oracle.topk_attention(q, kk, v, L, causal=causal)
    g = oracle.topk_attention_bwd(q, kk, v, dout, fwd["idx"])
    q64, k64, v64 = _f64(q), _f64(kk), _f64(v)
    out = torch.nn.functional.scaled_dot_product_attention(q64, k64, v64, scale=1.0, is_causal=causal)
    (out * dout.to(torch.float64)).sum().backward()
    np.testing.assert_allclose(g["dq"], q64.grad.numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(g["dk"], k64.grad.numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(g["dv"], v64.grad.numpy(), rtol=0, atol=1e-12)


def test_ffn_bwd_all_keys_equals_dense_ffn_gradient():
    """Eq. 3 with k = d_ff is the dense layer ReLU(x W1^T) W2; its gradient by autograd."""
    N, dm, dff = 17, 24, 40
    x, w1, w2 = workloads.ffn_inputs(N, dm, dff, dtype="bf16", seed=28)
    dout = _dout((N, dm), 29)
    fwd = oracle.ffn(x, w1, w2, dff)
    g = oracle.ffn_bwd(x, w1, w2, dout, fwd["idx"])
    x64, a64, b64 = _f64(x), _f64(w1), _f64(w2)
    out = torch.relu(x64 @ a64.T) @ b64
    (out * dout.to(torch.float64)).sum().backward()
    np.testing.assert_allclose(g["dx"], x64.grad.numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(g["dW1"], a64.grad.numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(g["dW2"], b64.grad.numpy(), rtol=0, atol=1e-12)


@pytest.mark.parametrize("act", [oracle.SOFTMAX, oracle.RELU])
def test_bwd_finite_differences(act):
    """Central differences of L = sum(dout * out) through the oracle's forward, kept set fixed."""
    B, H, Lq, Lk, d, k = 1, 2, 9, 14, 5, 4
    rng = np.random.default_rng(30)
    q = rng.standard_normal((B, H, Lq, d))
    kk = rng.standard_normal((B, H, Lk, d))
    v = rng.standard_normal((B, H, Lk, d))
    dout = rng.standard_normal((B, H, Lq, d))
    fwd = oracle.topk_attention(q, kk, v, k, act=act)
    idx = fwd["idx"]
    g = oracle.topk_attention_bwd(q, kk, v, dout, idx, act=act)
    if act == oracle.RELU:  # the ReLU kink must sit well away from every kept score
        assert np.min(np.abs(fwd["score"])) > 1e-3

    def loss(qq, kk2, vv):
        out, _ = oracle.eval_indices(qq, kk2, vv, idx, act=act)
        return float(np.sum(out * dout.reshape(-1, d)))

    h = 1e-6
    for name, arr, grad in (("q", q, g["dq"]), ("k", kk, g["dk"]), ("v", v, g["dv"])):
        for flat in rng.choice(arr.size, size=12, replace=False):
            pos = np.unravel_index(flat, arr.shape)
            args = {"q": q, "k": kk, "v": v}
            plus = {n: a.copy() for n, a in args.items()}
            minus = {n: a.copy() for n, a in args.items()}
            plus[name][pos] += h
            minus[name][pos] -= h
            fd = (loss(plus["q"], plus["k"], plus["v"]) - loss(minus["q"], minus["k"], minus["v"])) / (2 * h)
            assert abs(fd - grad[pos]) <= 1e-7 + 1e-6 * abs(fd), (name, pos, fd, grad[pos])


def test_bwd_softmax_invariants():
    B, H, Lq, Lk, d, k = 2, 3, 50, 70, 16, 12
    q, kk, v = workloads.attention_inputs(B, H, Lq, Lk, d, dtype="bf16", seed=31)
    dout = _dout((B, H, Lq, d), 32)
    fwd = oracle.topk_attention(q, kk, v, k)
    g = oracle.topk_attention_bwd(q, kk, v, dout, fwd["idx"])
    # the kept weights of each row sum to one: its score gradients sum to zero
    np.testing.assert_allclose(g["dk"].sum(axis=2), 0.0, atol=1e-11)
    np.testing.assert_allclose(g["dv"].sum(axis=2), dout.to(torch.float64).numpy().sum(axis=2), atol=1e-11)
    kept = _dense_mask(fwd["idx"], B, H, Lq, Lk).numpy().any(axis=2)  # [B,H,Lk]
    assert np.all(g["dk"][~kept] == 0) and np.all(g["dv"][~kept] == 0)
    assert np.all(np.abs(g["dv"][kept]).sum(axis=-1) > 0)


def test_ffn_bwd_negative_scores_give_no_gradient():
    """Kept FF scores that are all negative: ReLU is 0 there, so nothing flows back (Eq. 3)."""
    N, dm, dff, k = 6, 8, 20, 5
    x, w1, w2 = workloads.ffn_inputs(N, dm, dff, dtype="f32", seed=33)
    w1 = -torch.abs(w1)
    x = torch.abs(x)
    dout = _dout((N, dm), 34)
    fwd = oracle.ffn(x, w1, w2, k)
    assert np.all(fwd["score"] < 0)
    g = oracle.ffn_bwd(x, w1, w2, dout, fwd["idx"])
    assert np.all(g["dx"] == 0) and np.all(g["dW1"] == 0) and np.all(g["dW2"] == 0)
