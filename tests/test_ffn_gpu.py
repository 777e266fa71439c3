"""GPU parity: the top-k feed-forward layer (Eq. 3 with top-k) through the C ABI
against the CPU oracle, under the rules in _parity.py (ReLU activation,
fp32 output, bf16 inputs: outputs within 2e-2)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2106_06899_gb300 import topk as T
from paper_2106_06899_gb300 import workloads as W

from ._parity import check_rows

pytestmark = pytest.mark.gpu


def _run(x, w1, w2, topk):
    out, idx, score = T.ffn(x.cuda(), w1.cuda(), w2.cuda(), topk, return_indices=True)
    T.topk_check()
    return out.cpu(), idx.cpu(), score.cpu()


def _check(x, w1, w2, topk, rows=None):
    out, idx, score = _run(x, w1, w2, topk)
    rows = np.arange(x.shape[0]) if rows is None else np.asarray(rows)
    return check_rows(q=x[None, None], k=w1[None, None], v=w2[None, None], rows=rows,
                      gpu_out=out[rows].numpy(), gpu_idx=idx[rows].numpy(), gpu_score=score[rows].numpy(),
                      topk=topk, dtype="bf16", act=oracle.RELU)


def test_ffn_65k_sampled_rows():
    w = W.WORKLOADS["ffn_65k"]
    x, w1, w2 = W.make_inputs(w)
    rows = W.sample_rows(w.N, 48, seed=4).numpy()
    st = _check(x, w1, w2, w.topk, rows)
    assert st["rows"] == len(rows)


@pytest.mark.parametrize("topk", [1, 64, 512])
def test_ffn_ragged_all_rows(topk):
    # tokens and keys not multiples of the 128 x 256 tile
    x, w1, w2 = W.ffn_inputs(300, 128, 3000, seed=40 + topk)
    _check(x, w1, w2, topk)


def test_ffn_all_keys_is_dense_ffn():
    x, w1, w2 = W.ffn_inputs(130, 64, 256, seed=41)
    out, idx, _ = _run(x, w1, w2, 256)
    ref = torch.relu(x.double() @ w1.double().T) @ w2.double()
    assert (out.double() - ref).abs().max().item() <= 2e-2
    assert torch.equal(idx.sort(dim=1).values, torch.arange(256, dtype=torch.int32).expand(130, -1))


def test_ffn_wide_model_and_large_k():
    x, w1, w2 = W.ffn_inputs(200, 1024, 9000, seed=42)
    _check(x, w1, w2, 1000)


def test_ffn_key_permutation_equivariance():
    x, w1, w2 = W.ffn_inputs(128, 128, 2048, seed=43)
    perm = torch.randperm(2048, generator=torch.Generator().manual_seed(2))
    a_out, a_idx, _ = _run(x, w1, w2, 32)
    b_out, b_idx, _ = _run(x, w1[perm].contiguous(), w2[perm].contiguous(), 32)
    assert torch.allclose(a_out, b_out, atol=1e-5, rtol=0)
    assert torch.equal(perm[b_idx.long()].int(), a_idx)


def test_ffn_workspace_has_no_tokens_times_keys_term():
    # scratch is N x slices x list capacity (slices <= 64, capacity <= 6k + 1024 whatever d_ff is), a count
    # and a pooled-bound word per (token, slice), one bound word per token, plus the k kept keys of each
    # token (8 bytes each) for the gather
    for N in (128, 1000, 4096):
        for dff in (4096, 65536, 1 << 20):
            ws = T.topk_ffn_workspace_bytes(N, 1024, dff, 512)
            assert 0 < ws <= N * (64 * (6 * 512 + 1024) * 8 + 64 * 4 + 64 * 4 + 4 + 512 * 8) + 16
    assert T.topk_ffn_workspace_bytes(4096, 1024, 1 << 20, 512) < 4096 * (1 << 20)


def test_ffn_host_entry_matches_device_entry():
    x, w1, w2 = W.ffn_inputs(150, 128, 1500, seed=44)
    dev = T.ffn(x.cuda(), w1.cuda(), w2.cuda(), 40).cpu()
    out = torch.empty(150, 128, dtype=torch.float32).pin_memory()
    T.topk_ffn_fwd_host(x.pin_memory(), w1.pin_memory(), w2.pin_memory(), out, 40)
    assert torch.equal(out, dev)
