"""GPU parity of the backward pass (Sec. 2.2, "Improving efficiency through top-k
attention") through the C ABI against the fp64 oracle.

The backward pass takes the forward pass's cache, the kept indices and their
fp32 scores, as input.  Most tests build that cache without the CUDA path:
kept sets from the oracle's own forward pass or drawn at random (the backward
pass is defined for any kept set), with the scores the oracle computes for
them rounded to fp32.  Chain tests run the CUDA forward pass and then the
CUDA backward pass, and compare with the oracle's gradients for the oracle's
kept sets wherever the two sets agree.

Tolerance.  The CUDA path reads the bf16/fp32 inputs exactly and computes in
fp32; the oracle in fp64.  Each gradient element is a sum over at most
n + d products (n kept entries of a row or of a key, d the head size) of
terms bounded by the largest term of the tensor, so its fp32 rounding error
is at most about (n + d) * 2^-24 of the largest term, below 2e-5 of max|ref|
for n + d <= 300 (the fp32 rounding of the cached scores moves each weight
by a few units of 2^-24 more).  The tests allow 2e-5 * max|ref| per tensor
plus 2e-5 of the element itself; the errors measured on a GB300 are below
1e-6 of max|ref|.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2106_06899_gb300 import topk as T
from paper_2106_06899_gb300 import workloads as W

pytestmark = pytest.mark.gpu

RTOL = 2e-5


def _close(name, got, ref, rtol=RTOL):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    scale = float(np.max(np.abs(ref))) if ref.size else 0.0
    err = np.abs(got - ref)
    bound = rtol * scale + rtol * np.abs(ref)
    worst = float(np.max(err / np.maximum(bound, 1e-30))) if ref.size else 0.0
    assert np.all(err <= bound + 1e-30), f"{name}: max err {err.max():.3e}, scale {scale:.3e}, worst/bound {worst:.2f}"
    return float(err.max() / scale) if scale else 0.0


def _cache(q, k, v, idx, act):
    """A forward-pass cache for a kept set: its indices in the total order and their scores
    s_t = q_i . k_{j_t}, the oracle's fp64 values rounded to fp32 (-1 / -inf padded)."""
    _, sc, si = oracle.eval_indices(q, k, v, idx, act=act, return_idx=True)
    return torch.from_numpy(si), torch.from_numpy(sc.astype(np.float32))


def _attn_bwd_gpu(q, k, v, dout, idx, score):
    B, H, Lq, _ = q.shape
    K = idx.shape[-1]
    dq, dk, dv = T.attention_bwd(q.cuda(), k.cuda(), v.cuda(), dout.cuda(),
                                 idx.reshape(B, H, Lq, K).cuda(), score.reshape(B, H, Lq, K).cuda())
    T.topk_check()
    return dq.cpu().numpy(), dk.cpu().numpy(), dv.cpu().numpy()


def _compare_attn(g, ref):
    return [_close(n, g[i], ref["d" + n[1]]) for i, n in enumerate(("dq", "dk", "dv"))]


ATTN_CASES = [
    # dtype, B, H, Lq, Lk, d, k, kept-set recipe
    ("bf16", 1, 3, 300, 700, 64, 64, "oracle"),
    ("bf16", 2, 2, 257, 513, 128, 128, "oracle"),
    ("bf16", 1, 2, 190, 333, 64, 1, "oracle"),
    ("bf16", 1, 2, 96, 96, 64, 96, "oracle"),  # k = Lk: every key kept
    ("bf16", 2, 3, 211, 1000, 64, 48, "random"),
    ("bf16", 1, 2, 400, 3000, 128, 100, "hot"),  # a few keys kept by most rows: long runs, atomics
    ("f32", 1, 2, 200, 300, 64, 32, "oracle"),
    ("f32", 1, 2, 130, 260, 16, 20, "random"),
    ("f32", 2, 1, 150, 150, 32, 40, "oracle"),
    ("f32", 1, 1, 180, 500, 128, 256, "random"),
]


@pytest.mark.parametrize("dtype,B,H,Lq,Lk,d,k,sets", ATTN_CASES)
def test_attn_bwd_matches_oracle(dtype, B, H, Lq, Lk, d, k, sets):
    q, kk, v = W.attention_inputs(B, H, Lq, Lk, d, dtype=dtype, seed=40 + d + k)
    dout = W.grad_output((B, H, Lq, d), dtype=dtype, seed=41)
    if sets == "oracle":
        idx = torch.from_numpy(oracle.topk_attention(q, kk, v, k)["idx"])
    elif sets == "random":
        idx = W.kept_sets(B * H, Lq, Lk, k, seed=42, empty_frac=0.15)
    else:
        idx = W.kept_sets(B * H, Lq, Lk, k, seed=43, hot=12, hot_frac=0.9)
    cidx, score = _cache(q, kk, v, idx, oracle.SOFTMAX)
    g = _attn_bwd_gpu(q, kk, v, dout, cidx, score)
    ref = oracle.topk_attention_bwd(q, kk, v, dout, idx.numpy())
    errs = _compare_attn(g, ref)
    print(f"{dtype} B{B} H{H} Lq{Lq} Lk{Lk} d{d} k{k} {sets}: max err / scale dq {errs[0]:.1e} dk {errs[1]:.1e} "
          f"dv {errs[2]:.1e}")


def test_attn_bwd_causal_cache_with_short_rows():
    # causal kept sets: row i keeps min(i + 1, k) keys, the rest of its slots are -1
    B, H, L, d, k = 2, 2, 300, 128, 128
    q, kk, v = W.attention_inputs(B, H, L, L, d, dtype="bf16", seed=44)
    dout = W.grad_output((B, H, L, d), seed=45)
    idx = torch.from_numpy(oracle.topk_attention(q, kk, v, k, causal=True)["idx"])
    assert int((idx < 0).sum()) > 0
    g = _attn_bwd_gpu(q, kk, v, dout, *_cache(q, kk, v, idx, oracle.SOFTMAX))
    _compare_attn(g, oracle.topk_attention_bwd(q, kk, v, dout, idx.numpy()))


def test_attn_bwd_empty_cache_gives_zero_gradients():
    B, H, L, d, k = 1, 2, 64, 64, 8
    q, kk, v = W.attention_inputs(B, H, L, L, d, dtype="bf16", seed=46)
    dout = W.grad_output((B, H, L, d), seed=47)
    idx = torch.full((B * H * L, k), -1, dtype=torch.int32)
    score = torch.full((B * H * L, k), float("-inf"))
    dq, dk, dv = _attn_bwd_gpu(q, kk, v, dout, idx, score)
    assert not dq.any() and not dk.any() and not dv.any()


def test_attn_bwd_every_row_keeps_the_same_keys():
    # one run of entries per key spans many runs of the key pass: every flush is atomic
    B, H, Lq, Lk, d, k = 1, 1, 4096, 256, 64, 16
    q, kk, v = W.attention_inputs(B, H, Lq, Lk, d, dtype="bf16", seed=48)
    dout = W.grad_output((B, H, Lq, d), seed=49)
    idx = torch.arange(k, dtype=torch.int32).repeat(Lq, 1)
    g = _attn_bwd_gpu(q, kk, v, dout, *_cache(q, kk, v, idx, oracle.SOFTMAX))
    ref = oracle.topk_attention_bwd(q, kk, v, dout, idx.numpy())
    _compare_attn(g, ref)
    assert not g[1][0, 0, k:].any() and not g[2][0, 0, k:].any()


def _agreeing_rows_and_keys(gpu_idx, ref_idx, problems, Lq, Lk):
    """Rows whose kept sets agree, and keys whose gradient involves only agreeing rows."""
    gs = np.sort(np.where(gpu_idx < 0, np.iinfo(np.int32).max, gpu_idx), axis=1)
    rs = np.sort(np.where(ref_idx < 0, np.iinfo(np.int32).max, ref_idx), axis=1)
    agree = np.all(gs == rs, axis=1)
    key_ok = np.ones((problems, Lk), bool)
    for r in np.nonzero(~agree)[0]:
        p = r // Lq
        for j in np.concatenate([gpu_idx[r], ref_idx[r]]):
            if j >= 0:
                key_ok[p, j] = False
    return agree, key_ok


@pytest.mark.parametrize("causal,d,k", [(False, 64, 32), (True, 128, 128), (True, 64, 64)])
def test_attn_forward_then_backward_chain(causal, d, k):
    B, H, L = 1, 2, 640
    q, kk, v = W.attention_inputs(B, H, L, L, d, dtype="bf16", seed=50 + d)
    dout = W.grad_output((B, H, L, d), seed=51)
    out, idx, score = T.attention(q.cuda(), kk.cuda(), v.cuda(), k, causal=causal, return_indices=True)
    dq, dk, dv = T.attention_bwd(q.cuda(), kk.cuda(), v.cuda(), dout.cuda(), idx, score)
    T.topk_check()
    gpu_idx = idx.reshape(-1, k).cpu().numpy()
    ref_idx = oracle.topk_attention(q, kk, v, k, causal=causal)["idx"]
    ref = oracle.topk_attention_bwd(q, kk, v, dout, ref_idx)
    agree, key_ok = _agreeing_rows_and_keys(gpu_idx, ref_idx, B * H, L, L)
    assert agree.mean() > 0.99
    _close("dq", dq.cpu().numpy().reshape(-1, d)[agree], ref["dq"].reshape(-1, d)[agree])
    _close("dk", dk.cpu().numpy().reshape(B * H, L, d)[key_ok], ref["dk"].reshape(B * H, L, d)[key_ok])
    _close("dv", dv.cpu().numpy().reshape(B * H, L, d)[key_ok], ref["dv"].reshape(B * H, L, d)[key_ok])


def test_attn_bwd_long_65k_shape():
    # the long_65k forward workload's shape (B1 H12 L65536 d64 k64, low-rank inputs) with a random
    # cache in which 8 keys per head are kept by 30 % of the rows; every gradient element compared
    w = W.WORKLOADS["long_65k"]
    q, kk, v = W.make_inputs(w)
    dout = W.grad_output((w.B, w.H, w.Lq, w.d), seed=52)
    idx = W.kept_sets(w.B * w.H, w.Lq, w.Lk, w.topk, seed=53, hot=8, hot_frac=0.3)
    cidx, score = _cache(q, kk, v, idx, oracle.SOFTMAX)
    g = _attn_bwd_gpu(q, kk, v, dout, cidx, score)
    errs = _compare_attn(g, oracle.topk_attention_bwd(q, kk, v, dout, idx.numpy()))
    print(f"long_65k shape: max err / scale dq {errs[0]:.1e} dk {errs[1]:.1e} dv {errs[2]:.1e}")


# ---------------------------------------------------------------------------- feed-forward layer

def _ffn_bwd_gpu(x, w1, w2, dout, idx, score):
    dx, d1, d2 = T.ffn_bwd(x.cuda(), w1.cuda(), w2.cuda(), dout.cuda(), idx.cuda(), score.cuda())
    T.topk_check()
    return dx.cpu().numpy(), d1.cpu().numpy(), d2.cpu().numpy()


def _compare_ffn(g, ref):
    return [_close(n, g[i], ref[n]) for i, n in enumerate(("dx", "dW1", "dW2"))]


@pytest.mark.parametrize("N,dm,dff,k,sets", [
    (333, 256, 4096, 64, "oracle"),
    (128, 1024, 8192, 512, "oracle"),
    (200, 512, 3000, 100, "random"),  # about half the kept scores are <= 0: ReLU passes nothing back
    (96, 2048, 1024, 32, "random"),
    (64, 192, 700, 700, "oracle"),  # k = d_ff: the dense layer
])
def test_ffn_bwd_matches_oracle(N, dm, dff, k, sets):
    x, w1, w2 = W.ffn_inputs(N, dm, dff, seed=60 + k)
    dout = W.grad_output((N, dm), dtype="f32", seed=61)
    if sets == "oracle":
        idx = torch.from_numpy(oracle.ffn(x, w1, w2, k)["idx"])
    else:
        idx = W.kept_sets(1, N, dff, k, seed=62, empty_frac=0.1)
    cidx, score = _cache(x[None, None], w1[None, None], w2[None, None], idx, oracle.RELU)
    g = _ffn_bwd_gpu(x, w1, w2, dout, cidx, score)
    errs = _compare_ffn(g, oracle.ffn_bwd(x, w1, w2, dout, idx.numpy()))
    print(f"ffn N{N} dm{dm} dff{dff} k{k} {sets}: max err / scale dx {errs[0]:.1e} dW1 {errs[1]:.1e} "
          f"dW2 {errs[2]:.1e}")


def test_ffn_forward_then_backward_chain():
    N, dm, dff, k = 256, 512, 4096, 64
    x, w1, w2 = W.ffn_inputs(N, dm, dff, seed=63)
    dout = W.grad_output((N, dm), dtype="f32", seed=64)
    out, idx, score = T.ffn(x.cuda(), w1.cuda(), w2.cuda(), k, return_indices=True)
    dx, d1, d2 = T.ffn_bwd(x.cuda(), w1.cuda(), w2.cuda(), dout.cuda(), idx, score)
    T.topk_check()
    ref_idx = oracle.ffn(x, w1, w2, k)["idx"]
    ref = oracle.ffn_bwd(x, w1, w2, dout, ref_idx)
    agree, key_ok = _agreeing_rows_and_keys(idx.cpu().numpy(), ref_idx, 1, N, dff)
    assert agree.mean() > 0.9
    _close("dx", dx.cpu().numpy()[agree], ref["dx"][agree])
    _close("dW1", d1.cpu().numpy()[key_ok[0]], ref["dW1"][key_ok[0]])
    _close("dW2", d2.cpu().numpy()[key_ok[0]], ref["dW2"][key_ok[0]])


def test_ffn_bwd_ffn_65k_shape():
    # the ffn_65k forward workload's shape (N 4096, d_model 1024, d_ff 65536, k 512) with a random
    # cache in which 16 keys are kept by half the tokens; every gradient element compared
    w = W.WORKLOADS["ffn_65k"]
    x, w1, w2 = W.make_inputs(w)
    dout = W.grad_output((w.N, w.d_model), dtype="f32", seed=65)
    idx = W.kept_sets(1, w.N, w.d_ff, w.topk, seed=66, hot=16, hot_frac=0.5)
    cidx, score = _cache(x[None, None], w1[None, None], w2[None, None], idx, oracle.RELU)
    g = _ffn_bwd_gpu(x, w1, w2, dout, cidx, score)
    errs = _compare_ffn(g, oracle.ffn_bwd(x, w1, w2, dout, idx.numpy()))
    print(f"ffn_65k shape: max err / scale dx {errs[0]:.1e} dW1 {errs[1]:.1e} dW2 {errs[2]:.1e}")
