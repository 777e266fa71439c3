"""Seeded synthetic inputs shaped like the paper's workloads.

This module holds no arithmetic of the method: it only draws random tensors
(on the CPU, with ``torch.Generator``) in the shapes and distributions below.
Both the CUDA path's tests/benchmark and the CPU oracle read the very same
host tensors from here.

The shapes follow the paper's benchmark settings (Sec. 3): BERT-base
multi-head attention (12 heads of 64 dims, Sec. 3 "Multi-head attention
layer"), sequences up to 65,536 tokens with query chunks of 2^10 (Sec. 2.2
"Query chunking"), a causal decoder layer, and a feed-forward layer with
d_ff = 65,536 keys as in T5/UnifiedQA (Sec. 2.1 "Feed-forward as attention",
Sec. 4.3).  None of the paper's datasets or trained weights are used; these
random tensors stand in for them.

Distributions (the temperature lambda = sqrt(d) of Eq. 1 is folded into the
data, per the footnote to Eq. 1, by scaling both Q and K by d^-1/4):

* ``normal``  -- Q, K ~ N(0, 1) * d^-1/4, V ~ N(0, 1).
* ``lowrank`` -- Q = (G_q + s Z_q A) d^-1/4, K = (G_k + s Z_k A) d^-1/4 with
  G ~ N(0, 1) [L, d], Z ~ N(0, 1) [L, 8], A [8, d] with orthonormal rows drawn
  once per head, s = 2; V ~ N(0, 1).  The shared rank-8 part gives every
  score row a heavier upper tail than the isotropic case.
* ``ffn``     -- x ~ N(0, 1) [N, d_model]; W1, W2 ~ N(0, 1/d_model) [d_ff, d_model].
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import torch

LOWRANK_RANK = 8
LOWRANK_SCALE = 2.0


@dataclass(frozen=True)
class Workload:
    name: str
    kind: str  # "attn" or "ffn"
    dtype: str  # "f32" or "bf16"
    seed: int
    topk: int
    # attention
    B: int = 1
    H: int = 1
    Lq: int = 0
    Lk: int = 0
    d: int = 0
    chunk: int = 0
    causal: bool = False
    dist: str = "normal"
    # Eq. 2's general masks: key counts per batch (key padding), and the density of a random bit
    # mask shared by the heads of a batch (0 = none)
    kv_len: tuple = ()
    mask_p: float = 0.0
    # feed-forward
    N: int = 0
    d_model: int = 0
    d_ff: int = 0
    note: str = field(default="", compare=False)

    @property
    def rows(self) -> int:
        return self.B * self.H * self.Lq if self.kind == "attn" else self.N

    @property
    def tokens(self) -> int:
        return self.B * self.Lq if self.kind == "attn" else self.N

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


WORKLOADS = {
    "tiny_fp32": Workload("tiny_fp32", "attn", "f32", seed=0, topk=32, B=1, H=1, Lq=512, Lk=512, d=64,
                          chunk=128, note="tiny fp32 top-k attention"),
    "bert_base": Workload("bert_base", "attn", "bf16", seed=1, topk=64, B=8, H=12, Lq=512, Lk=512, d=64,
                          chunk=512, note="encoder-style BERT-base shape"),
    "bert_base_all_keys": Workload("bert_base_all_keys", "attn", "bf16", seed=1, topk=512, B=8, H=12, Lq=512,
                                   Lk=512, d=64, chunk=512, note="topk = Lk: must equal plain attention"),
    "long_65k": Workload("long_65k", "attn", "bf16", seed=2, topk=64, B=1, H=12, Lq=65536, Lk=65536, d=64,
                         chunk=1024, dist="lowrank", note="long-sequence top-64 attention, L = 65536"),
    "causal_16k": Workload("causal_16k", "attn", "bf16", seed=3, topk=128, B=2, H=16, Lq=16384, Lk=16384,
                           d=128, chunk=2048, causal=True, note="causal decoder-style, d = 128"),
    "ffn_65k": Workload("ffn_65k", "ffn", "bf16", seed=4, topk=512, N=4096, d_model=1024, d_ff=65536,
                        dist="ffn", note="top-k feed-forward, T5-large-like d_ff = 65536"),
    # Eq. 2's masks
    "decode_65k": Workload("decode_65k", "attn", "bf16", seed=5, topk=64, B=4, H=12, Lq=128, Lk=65536, d=64,
                           chunk=128, causal=True, dist="lowrank",
                           note="the last 128 positions against a 65,536-key cache, causal"),
    "bert_padded": Workload("bert_padded", "attn", "bf16", seed=6, topk=64, B=8, H=12, Lq=512, Lk=512, d=64,
                            chunk=512, kv_len=(512, 500, 448, 400, 320, 256, 128, 64),
                            note="BERT-base shape, batches padded to 512 keys"),
    "bert_masked": Workload("bert_masked", "attn", "bf16", seed=7, topk=64, B=8, H=12, Lq=512, Lk=512, d=64,
                            chunk=512, mask_p=0.5, note="BERT-base shape, random bit mask (half the pairs)"),
}


def mask_inputs(w: "Workload"):
    """(kv_len int32 [B] or None, boolean mask [B, 1, Lq, Lk] or None) of a workload, seeded."""
    kv = torch.tensor(w.kv_len, dtype=torch.int32) if w.kv_len else None
    mask = None
    if w.mask_p > 0:
        g = torch.Generator().manual_seed(int(w.seed) + 999)
        mask = torch.rand(w.B, 1, w.Lq, w.Lk, generator=g) < w.mask_p
    return kv, mask


def _torch_dtype(dtype: str) -> torch.dtype:
    return {"f32": torch.float32, "bf16": torch.bfloat16}[dtype]


def attention_inputs(B, H, Lq, Lk, d, *, dtype="bf16", seed=0, dist="normal"):
    """(q [B,H,Lq,d], k [B,H,Lk,d], v [B,H,Lk,d]) on the CPU in ``dtype``."""
    g = torch.Generator().manual_seed(int(seed))
    scale = d ** -0.25
    if dist == "normal":
        q = torch.randn(B, H, Lq, d, generator=g)
        k = torch.randn(B, H, Lk, d, generator=g)
    elif dist == "lowrank":
        r = min(LOWRANK_RANK, d)
        basis = torch.randn(H, d, r, generator=g, dtype=torch.float64)
        A = torch.linalg.qr(basis).Q.transpose(1, 2).to(torch.float32)  # [H, r, d], orthonormal rows
        q = torch.randn(B, H, Lq, d, generator=g)
        q += LOWRANK_SCALE * torch.randn(B, H, Lq, r, generator=g) @ A[None]
        k = torch.randn(B, H, Lk, d, generator=g)
        k += LOWRANK_SCALE * torch.randn(B, H, Lk, r, generator=g) @ A[None]
    elif dist == "integer":
        # small integers: every score is an exact integer in any precision, so
        # scores tie often and both sides see the same ties
        q = torch.randint(-2, 3, (B, H, Lq, d), generator=g).float()
        k = torch.randint(-2, 3, (B, H, Lk, d), generator=g).float()
        scale = 1.0
    else:
        raise ValueError(f"unknown distribution {dist!r}")
    v = torch.randn(B, H, Lk, d, generator=g)
    td = _torch_dtype(dtype)
    return (q * scale).to(td).contiguous(), (k * scale).to(td).contiguous(), v.to(td).contiguous()


def ffn_inputs(N, d_model, d_ff, *, dtype="bf16", seed=0, dist="ffn"):
    """(x [N,d_model], W1 [d_ff,d_model], W2 [d_ff,d_model]) on the CPU in ``dtype``.

    ``dist="integer"`` draws x and W1 from the integers -2..2 instead (W2 stays
    normal): every score is then an exact integer in any precision, so the
    k-th score is shared by many keys and both sides see the same ties."""
    g = torch.Generator().manual_seed(int(seed))
    td = _torch_dtype(dtype)
    std = 1.0 / math.sqrt(d_model)
    if dist == "ffn":
        x = torch.randn(N, d_model, generator=g)
        w1 = torch.randn(d_ff, d_model, generator=g) * std
    elif dist == "integer":
        x = torch.randint(-2, 3, (N, d_model), generator=g).float()
        w1 = torch.randint(-2, 3, (d_ff, d_model), generator=g).float()
    else:
        raise ValueError(f"unknown distribution {dist!r}")
    w2 = torch.randn(d_ff, d_model, generator=g) * std
    return x.to(td).contiguous(), w1.to(td).contiguous(), w2.to(td).contiguous()


def make_inputs(w: Workload):
    if w.kind == "attn":
        return attention_inputs(w.B, w.H, w.Lq, w.Lk, w.d, dtype=w.dtype, seed=w.seed, dist=w.dist)
    return ffn_inputs(w.N, w.d_model, w.d_ff, dtype=w.dtype, seed=w.seed)


def sample_rows(total: int, n: int, seed: int = 0) -> torch.Tensor:
    """n distinct row indices in [0, total), sorted, always including the first and last row."""
    n = min(n, total)
    g = torch.Generator().manual_seed(int(seed) + 12345)
    pick = torch.randperm(total, generator=g)[:n]
    pick[0] = 0
    if n > 1:
        pick[1] = total - 1
    return torch.unique(pick).sort().values


def grad_output(shape, *, dtype="bf16", seed=0) -> torch.Tensor:
    """dL/dout for the backward pass: N(0, 1) entries in ``dtype`` ("f32" or "bf16")."""
    g = torch.Generator().manual_seed(int(seed) + 777)
    return torch.randn(*shape, generator=g).to(_torch_dtype(dtype)).contiguous()


def kept_sets(problems: int, Lq: int, Lk: int, k: int, *, seed=0, hot: int = 0, hot_frac: float = 0.0,
              causal: bool = False, empty_frac: float = 0.0) -> torch.Tensor:
    """A kept-set cache [problems * Lq, k] int32 of distinct keys per row, -1 for empty slots.

    Drawn at random, not selected by score: the backward pass is defined for any kept
    set.  ``hot`` keys (0 .. hot-1) each enter a fraction ``hot_frac`` of the rows, so
    a few keys are kept by many rows, as the largest keys of a low-rank input are.
    With ``causal`` row i draws from keys 0 .. i only (all of them when i < k)."""
    g = torch.Generator().manual_seed(int(seed) + 4242)
    rows = problems * Lq
    n_valid = torch.full((rows,), Lk, dtype=torch.int64)
    if causal:
        n_valid = torch.clamp(torch.arange(rows) % Lq + 1, max=Lk)
    idx = torch.full((rows, k), -1, dtype=torch.int64)
    if hot:
        hot_in = torch.rand(rows, hot, generator=g) < hot_frac
        hot_in &= torch.arange(hot)[None, :] < n_valid[:, None]
    else:
        hot_in = torch.zeros(rows, 0, dtype=torch.bool)
    n_hot = hot_in.sum(1) if hot else torch.zeros(rows, dtype=torch.int64)
    # rows with few valid keys: a full permutation of them
    small = n_valid <= 4 * k
    for r in torch.nonzero(small).flatten().tolist():
        nv = int(n_valid[r])
        perm = torch.randperm(nv, generator=g)
        if hot:
            first = torch.nonzero(hot_in[r]).flatten()
            rest = perm[~torch.isin(perm, first)]
            perm = torch.cat([first, rest])
        take = min(k, nv)
        idx[r, :take] = perm[:take]
    # other rows: the hot keys they enter, then the rest of k from an arithmetic
    # progression hot + (base + t * stride) mod m over the m = n_valid - hot other keys,
    # with a random base and a random stride prime to m (so its first k terms differ)
    big = torch.nonzero(~small).flatten()
    if big.numel():
        m = n_valid[big] - hot
        base = (torch.rand(big.numel(), generator=g) * m).long()
        stride = 1 + (torch.rand(big.numel(), generator=g) * (m - 1)).long()
        bad = torch.gcd(stride, m) != 1
        while bool(bad.any()):
            stride = torch.where(bad, stride % (m - 1) + 1, stride)
            bad = torch.gcd(stride, m) != 1
        prog = torch.empty(big.numel(), k, dtype=torch.int64)
        x = base.clone()
        for t in range(k):  # x_t = (base + t stride) mod m, one add and one wrap per term
            prog[:, t] = x
            x += stride
            x -= m * (x >= m)
        prog += hot
        if hot:
            # the hot keys a row enters take its last slots
            filled = torch.zeros(big.numel(), dtype=torch.int64)
            hb = hot_in[big]
            rows_b = torch.arange(big.numel())
            for h in range(hot):
                sel = rows_b[hb[:, h]]
                prog[sel, k - 1 - filled[sel]] = h
                filled[sel] += 1
        idx[big] = prog
    if empty_frac > 0:
        idx[torch.rand(rows, k, generator=g) < empty_frac] = -1
    # the slot order within a row carries no meaning; shuffle the short rows' slots
    if bool(small.any()):
        sr = torch.nonzero(small).flatten()
        perm = torch.argsort(torch.rand(sr.numel(), k, generator=g), dim=1)
        idx[sr] = torch.gather(idx[sr], 1, perm)
    return idx.to(torch.int32).contiguous()
