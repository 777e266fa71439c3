"""GPU parity of Eq. 2's masks through the C ABI against the oracle (parity rules of _parity.py):

* causal with Lq < Lk (the queries are the last Lq positions: decoding against a key cache) on the
  tensor-core kernels, k = 64 (split kernel) and k = 128 (single-warp kernel), Lq from 1 up;
* per-batch key counts (key padding) on the tensor-core kernels, a batch with no key included;
* arbitrary bit masks, shared or per batch and head, on the CUDA-core kernel (bf16 and fp32),
  rows with no valid key included;
* all three together, and the backward pass for a masked forward pass's cache.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2106_06899_gb300 import topk as T
from paper_2106_06899_gb300 import workloads as W

from ._parity import check_rows
from .test_bwd_gpu import _agreeing_rows_and_keys

pytestmark = pytest.mark.gpu


def _run(q, k, v, topk, causal=False, kv_len=None, mask=None):
    kl = None if kv_len is None else torch.as_tensor(np.asarray(kv_len, np.int32)).cuda()
    mk = None if mask is None else torch.from_numpy(np.asarray(mask, bool)).cuda()
    out, idx, score = T.attention(q.cuda(), k.cuda(), v.cuda(), topk, causal=causal, return_indices=True,
                                  kv_len=kl, mask=mk)
    T.topk_check()
    return out.cpu(), idx.cpu(), score.cpu()


def _check(q, k, v, topk, dtype="bf16", causal=False, kv_len=None, mask=None, rows=None):
    out, idx, score = _run(q, k, v, topk, causal, kv_len, mask)
    B, H, Lq, d = q.shape
    rows = np.arange(B * H * Lq) if rows is None else np.asarray(rows)
    K = topk
    st = check_rows(q=q, k=k, v=v, rows=rows, gpu_out=out.float().reshape(-1, d)[rows].numpy(),
                    gpu_idx=idx.reshape(-1, K)[rows].numpy(), gpu_score=score.reshape(-1, K)[rows].numpy(),
                    topk=K, dtype=dtype, causal=causal, kv_len=kv_len, mask=mask)
    return st, out, idx


@pytest.mark.parametrize("Lq", [1, 7, 128, 300])
@pytest.mark.parametrize("d,k", [(64, 64), (128, 128)])
def test_causal_decode_tensor_cores(Lq, d, k):
    B, H, Lk = 2, 3, 2048
    q, kk, v = W.attention_inputs(B, H, Lq, Lk, d, seed=80 + Lq)
    st, _, _ = _check(q, kk, v, k, causal=True)
    assert st["exact_set_frac"] > 0.95, st


def test_decode_equals_last_rows_of_full_causal():
    # the last Lq queries against all keys, causal, give the same rows as the full causal problem
    B, H, L, d, k = 1, 2, 1024, 64, 64
    q, kk, v = W.attention_inputs(B, H, L, L, d, seed=85)
    full_out, full_idx, _ = _run(q, kk, v, k, causal=True)
    Lq = 200
    dec_out, dec_idx, _ = _run(q[:, :, L - Lq:].contiguous(), kk, v, k, causal=True)
    assert torch.equal(dec_idx, full_idx[:, :, L - Lq:])
    assert torch.equal(dec_out, full_out[:, :, L - Lq:])


@pytest.mark.parametrize("d,k", [(64, 64), (128, 128), (64, 100)])
def test_key_counts_tensor_cores(d, k):
    B, H, Lq, Lk = 4, 2, 256, 1500
    q, kk, v = W.attention_inputs(B, H, Lq, Lk, d, seed=86)
    kv_len = [1500, 777, 40, 0]  # 40 < k: those rows keep every valid key; 0: zeros
    st, out, idx = _check(q, kk, v, k, kv_len=kv_len)
    assert torch.all(out[3] == 0) and torch.all(idx[3] == -1)
    assert torch.all((idx[2] >= 0).sum(-1) == 40)
    assert st["exact_set_frac"] > 0.95, st


@pytest.mark.parametrize("dtype,d,k", [("bf16", 64, 32), ("bf16", 128, 64), ("f32", 64, 48), ("f32", 32, 200)])
@pytest.mark.parametrize("shape", ["full", "shared"])
def test_bit_mask(dtype, d, k, shape):
    B, H, Lq, Lk = 2, 3, 150, 777
    q, kk, v = W.attention_inputs(B, H, Lq, Lk, d, dtype=dtype, seed=87)
    rng = np.random.default_rng(88)
    mshape = (B, H, Lq, Lk) if shape == "full" else (1, 1, Lq, Lk)
    mask = rng.random(mshape) < 0.3
    mask[0, 0, 5] = False  # a row with no valid key
    mask[0, 0, 6] = False
    mask[0, 0, 6, 700:] = True  # a row with 77 valid keys: fewer than k when k = 200
    st, out, idx = _check(q, kk, v, k, dtype=dtype, mask=mask)
    assert torch.all(out[:, :, 5] == 0) if shape == "shared" else torch.all(out[0, 0, 5] == 0)
    assert st["exact_set_frac"] > 0.9, st


def test_all_masks_together():
    B, H, Lq, Lk, d, k = 2, 2, 100, 900, 64, 40
    q, kk, v = W.attention_inputs(B, H, Lq, Lk, d, seed=89)
    rng = np.random.default_rng(90)
    mask = rng.random((B, 1, Lq, Lk)) < 0.5
    st, _, _ = _check(q, kk, v, k, causal=True, kv_len=[900, 850], mask=mask)
    assert st["exact_set_frac"] > 0.95, st


def test_masked_forward_then_backward():
    # the cache of a masked forward pass feeds the backward pass; compare on rows whose kept sets agree
    B, H, Lq, Lk, d, k = 2, 2, 160, 640, 64, 32
    q, kk, v = W.attention_inputs(B, H, Lq, Lk, d, seed=91)
    kv_len = [640, 300]
    dout = W.grad_output((B, H, Lq, d), seed=92)
    _, idx, score = T.attention(q.cuda(), kk.cuda(), v.cuda(), k, causal=True, return_indices=True,
                                kv_len=torch.tensor(kv_len, dtype=torch.int32).cuda())
    dq, dk, dv = T.attention_bwd(q.cuda(), kk.cuda(), v.cuda(), dout.cuda(), idx, score)
    T.topk_check()
    ref_idx = oracle.topk_attention(q, kk, v, k, causal=True, kv_len=kv_len)["idx"]
    agree, key_ok = _agreeing_rows_and_keys(idx.reshape(-1, k).cpu().numpy(), ref_idx, B * H, Lq, Lk)
    assert agree.mean() > 0.99
    ref = oracle.topk_attention_bwd(q, kk, v, dout, ref_idx)
    pairs = (("dq", dq.cpu().numpy().reshape(-1, d)[agree], ref["dq"].reshape(-1, d)[agree]),
             ("dk", dk.cpu().numpy().reshape(B * H, Lk, d)[key_ok], ref["dk"].reshape(B * H, Lk, d)[key_ok]),
             ("dv", dv.cpu().numpy().reshape(B * H, Lk, d)[key_ok], ref["dv"].reshape(B * H, Lk, d)[key_ok]))
    for name, g, r in pairs:
        assert np.abs(g - r).max() <= 2e-5 * np.abs(r).max() + 1e-30, name
    assert not dk.cpu()[1, :, 300:].any() and not dv.cpu()[1, :, 300:].any()


@pytest.mark.parametrize("d,k", [(64, 200), (128, 300)])
def test_masks_on_reduced_row_units(d, k):
    # k above 137 runs on 64- or 32-row units: causal decode, key counts and key parts together
    B, H, Lq, Lk = 2, 2, 70, 1500
    q, kk, v = W.attention_inputs(B, H, Lq, Lk, d, seed=93)
    st, out, idx = _check(q, kk, v, k, causal=True, kv_len=[1500, 180])
    assert torch.all((idx[1] >= 0).sum(-1) == 180)  # every row of batch 1 keeps all its 180 keys
    assert st["exact_set_frac"] > 0.95, st
