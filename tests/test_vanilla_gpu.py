"""GPU parity of plain attention (Eq. 1 under Eq. 2's causal mask and key counts), the comparison
path, through the C ABI against the oracle's plain attention (pinned against SDPA).

The kernel rounds the softmax weights to bf16 before the P V product and writes bf16, so the
bf16 output tolerance of the top-k path (2e-2) applies.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2106_06899_gb300 import topk as T
from paper_2106_06899_gb300 import workloads as W

pytestmark = pytest.mark.gpu
TOL = 2e-2


def _run(q, k, v, causal=False, kv_len=None):
    kl = None if kv_len is None else torch.as_tensor(np.asarray(kv_len, np.int32)).cuda()
    out = T.vanilla_attention(q.cuda(), k.cuda(), v.cuda(), causal=causal, kv_len=kl)
    T.topk_check()
    return out.float().cpu().numpy().reshape(-1, q.shape[-1])


@pytest.mark.parametrize("B,H,Lq,Lk,d,causal", [
    (2, 3, 300, 700, 64, False),
    (1, 2, 257, 513, 128, False),
    (1, 2, 640, 640, 64, True),
    (2, 2, 7, 2048, 64, True),    # decode: the last 7 positions
    (1, 1, 1, 1001, 128, True),   # one query; a key count that is not a multiple of 8
    (3, 2, 129, 130, 64, False),  # ragged tiles on both sides
])
def test_vanilla_matches_oracle(B, H, Lq, Lk, d, causal):
    q, k, v = W.attention_inputs(B, H, Lq, Lk, d, seed=100 + Lq)
    got = _run(q, k, v, causal)
    ref = oracle.vanilla(q, k, v, causal=causal)
    err = np.abs(got - ref).max()
    assert err <= TOL, err


def test_vanilla_key_counts_and_empty_rows():
    B, H, Lq, Lk, d = 4, 2, 200, 900, 64
    q, k, v = W.attention_inputs(B, H, Lq, Lk, d, seed=110)
    kv_len = [900, 333, 5, 0]
    got = _run(q, k, v, kv_len=kv_len)
    ref = oracle.vanilla(q, k, v, kv_len=kv_len)
    assert np.abs(got - ref).max() <= TOL
    assert np.all(got.reshape(B, H, Lq, d)[3] == 0)


def test_vanilla_rescales_when_the_row_maximum_moves():
    # scores grow along the keys, so each row's maximum rises tile after tile (and by more than the
    # rescale margin): the running sum and O are rescaled many times
    B, H, Lq, Lk, d = 1, 2, 256, 4096, 64
    q, k, v = W.attention_inputs(B, H, Lq, Lk, d, dtype="f32", seed=111)
    ramp = torch.linspace(0.2, 6.0, Lk)[None, None, :, None]
    k = (k * ramp).to(torch.bfloat16)
    q = (q * 2).to(torch.bfloat16)
    v = v.to(torch.bfloat16)
    got = _run(q, k, v)
    ref = oracle.vanilla(q, k, v)
    assert np.abs(got - ref).max() <= TOL


def test_vanilla_equals_topk_with_every_key():
    # k = Lk keeps every key: the top-k path (CUDA-core kernel at k = 512) and the plain path agree
    w = W.WORKLOADS["bert_base_all_keys"]
    q, k, v = W.make_inputs(w)
    plain = _run(q, k, v)
    topk = T.attention(q.cuda(), k.cuda(), v.cuda(), w.topk).float().cpu().numpy().reshape(-1, w.d)
    assert np.abs(plain - topk).max() <= 2 * TOL


def test_vanilla_long_65k_sampled_rows():
    w = W.WORKLOADS["long_65k"].with_(H=2)
    q, k, v = W.make_inputs(w)
    got = _run(q, k, v)
    rows = W.sample_rows(w.rows, 512, seed=7).numpy()
    ref = oracle.vanilla(q, k, v, rows=rows)
    assert np.abs(got[rows] - ref).max() <= TOL


@pytest.mark.parametrize("N,dm,dff,chunk", [
    (333, 256, 4096, 1024),
    (128, 1024, 65536, 16384),
    (200, 512, 3000, 1024),   # a last slice of 952 keys
    (64, 192, 700, 700),      # one slice
])
def test_dense_ffn_matches_oracle(N, dm, dff, chunk):
    # the hidden activations H = ReLU(x W1^T) are rounded to bf16 (8-bit significand: relative error
    # at most 2^-8 under round-to-nearest) before the second product, so an output element can be off
    # by up to 2^-8 sum_j H_j |W2_j|, plus the fp32 sums (1e-5); that sum is the dense layer applied
    # to |W2| (the oracle's, exact)
    x, w1, w2 = W.ffn_inputs(N, dm, dff, seed=120 + N)
    out = T.vanilla_ffn(x.cuda(), w1.cuda(), w2.cuda(), chunk)
    T.topk_check()
    ref = oracle.ffn_dense(x, w1, w2)
    scale = oracle.ffn_dense(x, w1, w2.abs())
    err = np.abs(out.cpu().numpy() - ref)
    assert np.all(err <= 2.0 ** -8 * scale + 1e-5), float((err / (2.0 ** -8 * scale + 1e-5)).max())


def test_dense_ffn_equals_topk_ffn_with_every_key():
    # k = d_ff keeps every key: both paths compute the dense layer (each within its own bound)
    N, dm, dff = 96, 256, 1024
    x, w1, w2 = W.ffn_inputs(N, dm, dff, seed=130)
    dense = T.vanilla_ffn(x.cuda(), w1.cuda(), w2.cuda(), 512).cpu().numpy()
    topk = T.ffn(x.cuda(), w1.cuda(), w2.cuda(), dff).cpu().numpy()
    ref = oracle.ffn_dense(x, w1, w2)
    scale = oracle.ffn_dense(x, w1, w2.abs())
    assert np.all(np.abs(dense - ref) <= 2.0 ** -8 * scale + 1e-5)
    assert np.abs(topk - ref).max() <= TOL
