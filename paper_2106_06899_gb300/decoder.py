"""A decoder stack composed of the library's calls: the 12-layer decoder of the paper's
benchmarks (Sec. 3, "12-layer decoder"), trained end to end.

Every layer is pre-LayerNorm causal self-attention followed by a feed-forward layer, each with
a residual connection.  The attention is top-k attention (Eq. 4) through the C ABI, forward with
the kept (index, score) cache and backward from that cache (Sec. 2.2); the feed-forward layer is
either the top-k FF layer (Eq. 3 with top-k) through the C ABI, forward and backward, or the
dense layer.  The projections, LayerNorms and the dense FF layer are ordinary PyTorch operations:
they are the model around the method, not part of it.  The temperature of Eq. 1 is folded into Q
(footnote to Eq. 1).
"""
from __future__ import annotations

import torch

from . import topk as T


class TopKAttentionFunction(torch.autograd.Function):
    """Top-k attention with the paper's caching: the forward pass keeps q, k, v and the kept
    (index, score) lists, O(L k) per head, and the backward pass recomputes only the activation."""

    @staticmethod
    def forward(ctx, q, k, v, topk: int, causal: bool):
        out, idx, score = T.attention(q, k, v, topk, causal=causal, return_indices=True)
        ctx.save_for_backward(q, k, v, idx, score)
        return out

    @staticmethod
    def backward(ctx, dout):
        q, k, v, idx, score = ctx.saved_tensors
        dq, dk, dv = T.attention_bwd(q, k, v, dout.to(q.dtype).contiguous(), idx, score)
        return dq.to(q.dtype), dk.to(k.dtype), dv.to(v.dtype), None, None


class TopKFFNFunction(torch.autograd.Function):
    """The top-k FF layer with the same caching: x [N, d_model], W1/W2 [d_ff, d_model] (bf16)."""

    @staticmethod
    def forward(ctx, x, w1, w2, topk: int):
        out, idx, score = T.ffn(x, w1, w2, topk, return_indices=True)
        ctx.save_for_backward(x, w1, w2, idx, score)
        return out

    @staticmethod
    def backward(ctx, dout):
        x, w1, w2, idx, score = ctx.saved_tensors
        dx, d1, d2 = T.ffn_bwd(x, w1, w2, dout.float().contiguous(), idx, score)
        return dx.to(x.dtype), d1.to(w1.dtype), d2.to(w2.dtype), None


class DecoderLayer(torch.nn.Module):
    def __init__(self, d_model: int, heads: int, d_ff: int, topk: int | None, ffn_topk: int | None,
                 dtype=torch.bfloat16, device="cuda"):
        super().__init__()
        self.h, self.dh = heads, d_model // heads
        self.topk, self.ffn_topk = topk, ffn_topk
        kw = dict(dtype=dtype, device=device)
        self.ln1 = torch.nn.LayerNorm(d_model, **kw)
        self.ln2 = torch.nn.LayerNorm(d_model, **kw)
        self.qkv = torch.nn.Linear(d_model, 3 * d_model, bias=False, **kw)
        self.proj = torch.nn.Linear(d_model, d_model, bias=False, **kw)
        # FF keys and values are the rows of W1 and W2 (Sec. 2.1)
        self.w1 = torch.nn.Parameter(torch.randn(d_ff, d_model, **kw) * d_model ** -0.5)
        self.w2 = torch.nn.Parameter(torch.randn(d_ff, d_model, **kw) * d_ff ** -0.5)

    def attention(self, q, k, v):
        if self.topk is None:  # plain causal attention (PyTorch), the comparison
            return torch.nn.functional.scaled_dot_product_attention(q, k, v, is_causal=True, scale=1.0)
        return TopKAttentionFunction.apply(q, k, v, self.topk, True)

    def feed_forward(self, h):
        if self.ffn_topk is None:
            return torch.relu(h @ self.w1.t()) @ self.w2
        return TopKFFNFunction.apply(h.contiguous(), self.w1, self.w2, self.ffn_topk).to(h.dtype)

    def forward(self, x):
        B, L, D = x.shape
        qkv = self.qkv(self.ln1(x)).view(B, L, 3, self.h, self.dh).permute(2, 0, 3, 1, 4)
        q = (qkv[0] * self.dh ** -0.5).contiguous()  # Eq. 1's temperature folded into Q
        k, v = qkv[1].contiguous(), qkv[2].contiguous()
        a = self.attention(q, k, v)
        x = x + self.proj(a.transpose(1, 2).reshape(B, L, D))
        f = self.feed_forward(self.ln2(x).reshape(B * L, D))
        return x + f.view(B, L, D)


class Decoder(torch.nn.Module):
    """n_layers decoder layers over d_model features; topk / ffn_topk None selects the plain
    attention / the dense FF layer."""

    def __init__(self, n_layers=12, d_model=768, heads=12, d_ff=3072, topk: int | None = 64,
                 ffn_topk: int | None = None, dtype=torch.bfloat16, device="cuda"):
        super().__init__()
        self.layers = torch.nn.ModuleList(
            DecoderLayer(d_model, heads, d_ff, topk, ffn_topk, dtype, device) for _ in range(n_layers))
        self.norm = torch.nn.LayerNorm(d_model, dtype=dtype, device=device)

    def forward(self, x):
        for layer in self.layers:
            x = layer(x)
        return self.norm(x)
