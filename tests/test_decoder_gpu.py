"""The 12-layer decoder composition (Sec. 3) built from the library's calls, on the GPU.

With k = L (every key kept) top-k attention is plain causal attention, and with k = d_ff the top-k
FF layer is the dense one, so the composed decoder -- forward and every parameter gradient -- must
compute what the same decoder written with PyTorch's scaled_dot_product_attention and matrix
products computes (a library reference, independent of this code).  The weights and activations
are bf16, whose rounding alone moves a two-layer network's gradients by several per cent, so both
bf16 decoders are measured against the same decoder in fp32: the composition must be about as
close to it as the plain bf16 decoder is.
"""
import pytest
import torch

from paper_2106_06899_gb300.decoder import Decoder

pytestmark = pytest.mark.gpu


def _rel(a, b):
    return ((a.float() - b.float()).abs().max() / b.float().abs().max()).item()


def _run(models, xs, g):
    res = []
    for m, x in zip(models, xs):
        y = m(x)
        (y.float() * g.float()).sum().backward()
        res.append((y.detach(), {n: p.grad for n, p in m.named_parameters()}))
    return res


def test_decoder_fp32_with_every_key_equals_the_plain_decoder():
    # fp32 end to end (the attention runs on the CUDA-core kernel, the FF layer is dense): the composed
    # forward and backward must match PyTorch's to fp32 rounding
    torch.manual_seed(0)
    B, L, D, H, F, layers = 2, 256, 256, 4, 512, 2
    topk_model = Decoder(layers, D, H, F, topk=L, ffn_topk=None, dtype=torch.float32)
    plain_model = Decoder(layers, D, H, F, topk=None, ffn_topk=None, dtype=torch.float32)
    plain_model.load_state_dict(topk_model.state_dict())
    x = torch.randn(B, L, D, device="cuda")
    g = torch.randn(B, L, D, device="cuda")
    (yt, gt), (yp, gp) = _run((topk_model, plain_model), (x, x), g)
    assert _rel(yt, yp) <= 1e-4
    # a ReLU pre-activation within rounding of 0 can take the other side in one of the two runs; the
    # flipped unit moves its token's gradient, and through it every earlier gradient, by up to about
    # 1e-2 of the largest element (a wrong composition is off by O(1))
    for n in gp:
        assert _rel(gt[n], gp[n]) <= 1e-2, n


def test_attention_function_matches_sdpa_autograd():
    # the autograd wrapper alone (no ReLU downstream): forward and the three input gradients
    from paper_2106_06899_gb300.decoder import TopKAttentionFunction

    torch.manual_seed(3)
    B, H, L, d = 2, 3, 384, 64
    q, k, v = (torch.randn(B, H, L, d, device="cuda") * (d ** -0.25) for _ in range(3))
    g = torch.randn(B, H, L, d, device="cuda")
    qs, ks, vs = (t.clone().requires_grad_() for t in (q, k, v))
    ref = torch.nn.functional.scaled_dot_product_attention(qs, ks, vs, is_causal=True, scale=1.0)
    (ref * g).sum().backward()
    qt, kt, vt = (t.clone().requires_grad_() for t in (q, k, v))
    out = TopKAttentionFunction.apply(qt, kt, vt, L, True)
    (out * g).sum().backward()
    assert _rel(out, ref) <= 1e-5
    for a, b in ((qt.grad, qs.grad), (kt.grad, ks.grad), (vt.grad, vs.grad)):
        assert _rel(a, b) <= 1e-4


def test_decoder_bf16_with_every_key_and_topk_ffn_matches_the_plain_decoder():
    # bf16 weights and activations, the FF layer top-k with k = d_ff: bf16 rounding alone moves a
    # two-layer network's gradients by several per cent, so both bf16 decoders are measured against
    # the decoder in fp32 and the composition must be about as close to it as the plain one
    torch.manual_seed(0)
    B, L, D, H, F, layers = 2, 256, 256, 4, 512, 2
    topk_model = Decoder(layers, D, H, F, topk=L, ffn_topk=F)
    plain_model = Decoder(layers, D, H, F, topk=None, ffn_topk=None)
    plain_model.load_state_dict(topk_model.state_dict())
    ref = Decoder(layers, D, H, F, topk=None, ffn_topk=None, dtype=torch.float32)
    ref.load_state_dict({k: v.float() for k, v in topk_model.state_dict().items()})
    x = torch.randn(B, L, D, device="cuda", dtype=torch.bfloat16)
    g = torch.randn(B, L, D, device="cuda", dtype=torch.bfloat16)
    (yt, gt), (yp, gp), (yr, gr) = _run((topk_model, plain_model, ref), (x, x, x.float()), g)
    assert _rel(yt, yr) <= max(2 * _rel(yp, yr), 1e-2)
    for n in gr:
        e_topk, e_plain = _rel(gt[n], gr[n]), _rel(gp[n], gr[n])
        assert e_topk <= max(2 * e_plain, 3e-2), (n, e_topk, e_plain)


def test_decoder_top64_trains():
    torch.manual_seed(1)
    B, L, D, H, F, layers = 1, 2048, 256, 4, 1024, 2
    m = Decoder(layers, D, H, F, topk=64, ffn_topk=None)
    x = torch.randn(B, L, D, device="cuda", dtype=torch.bfloat16)
    y = m(x)
    loss = y.float().pow(2).mean()
    loss.backward()
    assert torch.isfinite(loss)
    for n, p in m.named_parameters():
        assert p.grad is not None and torch.isfinite(p.grad.float()).all(), n
        assert p.grad.float().abs().sum() > 0, n


def test_decoder_top64_with_topk_ffn_trains():
    torch.manual_seed(2)
    B, L, D, H, F, layers = 1, 1024, 256, 4, 4096, 2
    m = Decoder(layers, D, H, F, topk=64, ffn_topk=256)
    x = torch.randn(B, L, D, device="cuda", dtype=torch.bfloat16)
    y = m(x)
    y.float().pow(2).mean().backward()
    for n, p in m.named_parameters():
        assert p.grad is not None and torch.isfinite(p.grad.float()).all(), n
