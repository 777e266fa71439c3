"""The C-ABI library loads and exports every symbol include/topk_attention.h declares,
and rejects bad arguments before launching anything (CPU only: no compute call runs)."""
import ctypes
import os
import re

import pytest

from paper_2106_06899_gb300 import build
from paper_2106_06899_gb300 import topk as T

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    text = open(os.path.join(ROOT, "include", "topk_attention.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(topk_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    build.build_library()
    return T.lib()


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert "topk_attn_fwd" in names and "topk_ffn_fwd" in names
    for n in names:
        assert hasattr(lib, n), n


def test_error_strings(lib):
    for code in (0, -1, -2, -3, -4, -5, -6):
        assert T.error_string(code)
    assert T.error_string(-99) == "unknown error code"


def _attn(lib, **kw):
    a = dict(q=16, k=16, v=16, out=16, B=1, H=1, Lq=8, Lk=8, d=64, topk=4, chunk=8, causal=0, dtype=1)
    a.update(kw)
    return lib.topk_attn_fwd(a["q"], a["k"], a["v"], a["out"], a["B"], a["H"], a["Lq"], a["Lk"], a["d"],
                             a["topk"], a["chunk"], a["causal"], a["dtype"], None)


@pytest.mark.parametrize("kw,code", [
    (dict(q=None), -1), (dict(out=None), -1), (dict(B=0), -1), (dict(Lk=-1), -1), (dict(topk=0), -1),
    (dict(topk=9), -1), (dict(chunk=0), -1), (dict(causal=1, Lq=9, topk=2), -1), (dict(causal=2), -1),
    (dict(dtype=7), -1), (dict(d=96), -2), (dict(dtype=0, d=48), -2), (dict(topk=600, Lk=1000), -2),
    (dict(q=24), -2),
])
def test_attention_argument_errors(lib, kw, code):
    assert _attn(lib, **kw) == code


def test_ffn_argument_errors(lib):
    f = lib.topk_ffn_fwd
    assert f(None, 16, 16, 16, 4, 64, 128, 8, None) == -1
    assert f(16, 16, 16, 16, 4, 64, 128, 0, None) == -1
    assert f(16, 16, 16, 16, 4, 64, 128, 129, None) == -1
    assert f(16, 16, 16, 16, 4, 100, 128, 8, None) == -2
    assert f(16, 16, 16, 16, 4, 64, 4096, 2000, None) == -2


def test_attention_workspace_does_not_grow_with_the_sequence():
    # the tcgen05 split kernel parks each work unit's kept keys for its epilogue warps: per CTA (at most
    # one per SM) 4 heap warps x 2 slots x k keys x 32 rows x 8 bytes, plus a count per row; nothing per
    # query row or key, so the scratch is the same at 8K, 64K and 1M tokens
    sizes = {T.topk_attn_workspace_bytes(1, 12, L, L, 64, 64, 1024, 1) for L in (8192, 65536, 1 << 20)}
    assert len(sizes) == 1
    (ws,) = sizes
    assert 0 < ws <= 1024 * (4 * 2 * 64 * 32 * 8 + 4 * 2 * 32 * 4)
    # fp32 inputs and k above the tensor path's limit run the SIMT kernel, which needs none
    assert T.topk_attn_workspace_bytes(1, 12, 65536, 65536, 64, 64, 1024, 0) == 0
    assert T.topk_attn_workspace_bytes(1, 12, 4096, 4096, 64, 256, 1024, 1) == 0
    # invalid arguments report 0
    assert T.topk_attn_workspace_bytes(1, 12, 4096, 4096, 64, 0, 1024, 1) == 0


def _attn_bwd(lib, **kw):
    a = dict(q=16, k=16, v=16, dout=16, idx=16, score=16, dq=16, dk=16, dv=16, B=1, H=1, Lq=8, Lk=8, d=64,
             topk=4, dtype=1)
    a.update(kw)
    return lib.topk_attn_bwd(a["q"], a["k"], a["v"], a["dout"], a["idx"], a["score"], a["dq"], a["dk"], a["dv"],
                             a["B"], a["H"], a["Lq"], a["Lk"], a["d"], a["topk"], a["dtype"], None)


@pytest.mark.parametrize("kw,code", [
    (dict(q=None), -1), (dict(dout=None), -1), (dict(idx=None), -1), (dict(dv=None), -1), (dict(B=0), -1),
    (dict(topk=0), -1), (dict(topk=9), -1), (dict(dtype=5), -1), (dict(d=96), -2), (dict(dtype=0, d=48), -2),
    (dict(topk=3000, Lk=4000), -2), (dict(dq=24), -2), (dict(idx=18), -2),
    (dict(B=1 << 16, H=1 << 10, Lq=64, topk=4, Lk=8), -2),
])
def test_attention_backward_argument_errors(lib, kw, code):
    assert _attn_bwd(lib, **kw) == code


def test_ffn_backward_argument_errors(lib):
    f = lib.topk_ffn_bwd
    ok = [16] * 9
    assert f(*([None] + ok[1:]), 4, 64, 128, 8, None) == -1
    assert f(*ok, 4, 64, 128, 0, None) == -1
    assert f(*ok, 4, 64, 128, 129, None) == -1
    assert f(*ok, 4, 100, 128, 8, None) == -2
    assert f(*ok, 4, 4096, 128, 8, None) == -2
    assert f(*(ok[:6] + [24] + ok[7:]), 4, 64, 128, 8, None) == -2


def test_backward_scratch_is_linear_in_the_cache():
    # rank + entry per cached (row, slot): 20 bytes; count + offset per key: 8 bytes; nothing per (query, key)
    def attn(L, k):
        return T.topk_attn_bwd_workspace_bytes(1, 12, L, L, 64, k, 1)
    for L in (8192, 65536):
        ws = attn(L, 64)
        entries, keys = 12 * L * 64, 12 * L
        assert entries * 20 + keys * 8 <= ws <= entries * 20 + keys * 8 + 5 * 256 + 4 * (keys // 4096 + 1)
    # doubling L doubles the growth (up to the 256-byte alignment of the parts): linear, no L^2 term
    assert abs((attn(65536, 64) - attn(32768, 64)) - 2 * (attn(32768, 64) - attn(16384, 64))) <= 2048
    f = T.topk_ffn_bwd_workspace_bytes
    # FF: also the partial dot products per 256-column chunk of d_model (4 chunks at 1024)
    assert 4096 * 512 * 36 <= f(4096, 1024, 65536, 512) <= 4096 * 512 * 36 + 65536 * 8 + 4096
    assert f(4096, 4096, 65536, 512) == 0 and attn(1024, 0) == 0


def test_masked_attention_argument_errors(lib):
    f = lib.topk_attn_fwd_masked

    def call(causal=0, kv_len=None, mask=None, mbs=0, mhs=0, Lq=8, Lk=8):
        return f(16, 16, 16, 16, 1, 1, Lq, Lk, 64, 4, 8, causal, kv_len, mask, mbs, mhs, 1, None, None, None)

    assert call(mbs=-1, mask=16) == -1
    assert call(mhs=-4, mask=16) == -1
    assert call(causal=1, Lq=9) == -1
    assert call(mask=18) == -2      # not 4-byte aligned
    assert call(kv_len=17) == -2


def test_vanilla_attention_argument_errors(lib):
    f = lib.topk_vanilla_attn_fwd

    def call(q=16, B=1, H=1, Lq=8, Lk=8, d=64, chunk=8, causal=0, kv_len=None, dtype=1):
        return f(q, 16, 16, 16, B, H, Lq, Lk, d, chunk, causal, kv_len, dtype, None)

    assert call(q=None) == -1 and call(Lk=0) == -1 and call(chunk=0) == -1 and call(dtype=3) == -1
    assert call(causal=1, Lq=9) == -1
    assert call(dtype=0) == -2 and call(d=96) == -2 and call(q=24) == -2
    assert call(B=300, H=300) == -2  # more than 65535 (batch, head) problems
    # scratch: V transposed, keys rounded up to a multiple of 8
    assert T.topk_vanilla_attn_workspace_bytes(2, 3, 100, 1001, 64, 1) == 2 * 3 * 64 * 1008 * 2
    assert T.topk_vanilla_attn_workspace_bytes(2, 3, 100, 1001, 64, 0) == 0


def test_dense_ffn_argument_errors(lib):
    f = lib.topk_vanilla_ffn_fwd
    assert f(None, 16, 16, 16, 4, 64, 128, 64, None) == -1
    assert f(16, 16, 16, 16, 4, 64, 128, 0, None) == -1
    assert f(16, 16, 16, 16, 4, 60, 128, 64, None) == -2   # d_model not a multiple of 8
    assert f(16, 16, 16, 16, 4, 64, 128, 60, None) == -2   # slice not a multiple of 8
    assert f(24, 16, 16, 16, 4, 64, 128, 64, None) == -2
    assert T.topk_vanilla_ffn_workspace_bytes(4096, 1024, 65536, 16384) == 4096 * 16384 * 2
    assert T.topk_vanilla_ffn_workspace_bytes(4096, 1024, 1000, 16384) == 4096 * 1000 * 2
