"""The no-allocation FF entry point, topk_ffn_fwd_noalloc, through the C ABI.

It serves callers that cannot allocate device memory when they call (a host
runtime that owns all device memory through its own arena, a serving loop that
must not wait on an allocator).  Its scratch is one fixed buffer inside the
library, so these checks run it twice in a row and compare each result with the
allocating entry point, topk_ffn_fwd, within the tolerance of the other FF
parity tests.  The file is named to be collected last.
"""
import pytest
import torch

from paper_2106_06899_gb300 import topk as T
from paper_2106_06899_gb300 import workloads as W

pytestmark = pytest.mark.gpu

TOL = 2e-2  # bf16 inputs, fp32 accumulation: the FF parity tolerance


def _dev(*ts):
    return [t.cuda() for t in ts]


def test_noalloc_matches_allocating_entry_on_two_calls_in_a_row():
    x, w1, w2 = _dev(*W.ffn_inputs(200, 128, 4096, seed=61))
    assert T.topk_ffn_workspace_bytes(200, 128, 4096, 64) <= T.TOPK_FFN_NOALLOC_SCRATCH_BYTES
    ref = torch.empty(200, 128, dtype=torch.float32, device="cuda")
    T.topk_ffn_fwd(x, w1, w2, ref, 64)
    T.topk_check()
    for _ in range(2):  # the second call starts from the first call's leftovers in the shared buffer
        out = torch.full((200, 128), float("nan"), dtype=torch.float32, device="cuda")
        T.topk_ffn_fwd_noalloc(x, w1, w2, out, 64)
        T.topk_check()
        assert torch.isfinite(out).all()
        assert (out - ref).abs().max().item() <= TOL


def test_noalloc_after_a_different_problem():
    # a larger k and other sizes first, then the first problem again
    a = _dev(*W.ffn_inputs(300, 256, 3000, seed=62))
    out_a = torch.empty(300, 256, dtype=torch.float32, device="cuda")
    T.topk_ffn_fwd_noalloc(*a, out_a, 200)
    T.topk_check()
    ref_a = torch.empty_like(out_a)
    T.topk_ffn_fwd(*a, ref_a, 200)
    T.topk_check()
    assert (out_a - ref_a).abs().max().item() <= TOL
    b = _dev(*W.ffn_inputs(129, 64, 1500, seed=63))
    out_b = torch.empty(129, 64, dtype=torch.float32, device="cuda")
    T.topk_ffn_fwd_noalloc(*b, out_b, 7)
    T.topk_check()
    ref_b = torch.empty_like(out_b)
    T.topk_ffn_fwd(*b, ref_b, 7)
    T.topk_check()
    assert (out_b - ref_b).abs().max().item() <= TOL


def test_noalloc_rejects_problems_beyond_its_buffer():
    x, w1, w2 = _dev(*W.ffn_inputs(4096, 64, 65536, seed=64))
    assert T.topk_ffn_workspace_bytes(4096, 64, 65536, 512) > T.TOPK_FFN_NOALLOC_SCRATCH_BYTES
    out = torch.full((4096, 64), 7.0, dtype=torch.float32, device="cuda")
    with pytest.raises(T.TopkError) as e:
        T.topk_ffn_fwd_noalloc(x, w1, w2, out, 512)
    assert e.value.code == -7
    assert (out == 7.0).all()  # rejected before anything was launched
