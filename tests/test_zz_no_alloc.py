"""The no-allocation FF entry point, topk_ffn_fwd_noalloc, through the C ABI.

It serves callers that cannot allocate device memory when they call (a host
runtime that owns all device memory through its own arena, a serving loop that
must not wait on an allocator).  Its scratch is one fixed buffer inside the
library, shared by every call, so these checks run it twice in a row and after
a different problem, and require the same bits as the allocating entry point,
topk_ffn_fwd (the FF path is deterministic), plus the oracle's parity rules
once.  The file is named to be collected last.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2106_06899_gb300 import topk as T
from paper_2106_06899_gb300 import workloads as W

from ._parity import check_rows

pytestmark = pytest.mark.gpu


def _dev(*ts):
    return [t.cuda() for t in ts]


def _reference(x, w1, w2, topk):
    ref = torch.empty(x.shape[0], x.shape[1], dtype=torch.float32, device="cuda")
    T.topk_ffn_fwd(x, w1, w2, ref, topk)
    T.topk_check()
    return ref


def test_noalloc_matches_allocating_entry_on_two_calls_in_a_row():
    host = W.ffn_inputs(200, 128, 4096, seed=61)
    x, w1, w2 = _dev(*host)
    assert T.topk_ffn_workspace_bytes(200, 128, 4096, 64) <= T.TOPK_FFN_NOALLOC_SCRATCH_BYTES
    ref = _reference(x, w1, w2, 64)
    for _ in range(2):  # the second call starts from the first call's leftovers in the shared buffer
        out = torch.full((200, 128), float("nan"), dtype=torch.float32, device="cuda")
        T.topk_ffn_fwd_noalloc(x, w1, w2, out, 64)
        T.topk_check()
        assert torch.equal(out, ref)
    # and against the oracle, under the parity rules of the other FF tests
    _, idx, score = T.ffn(x, w1, w2, 64, return_indices=True)
    rows = np.arange(200)
    check_rows(q=host[0][None, None], k=host[1][None, None], v=host[2][None, None], rows=rows,
               gpu_out=out.cpu().numpy(), gpu_idx=idx.cpu().numpy(), gpu_score=score.cpu().numpy(), topk=64,
               dtype="bf16", act=oracle.RELU)


def test_noalloc_after_a_different_problem():
    # a larger k and other sizes first, then a smaller problem: stale scratch must not leak through
    a = _dev(*W.ffn_inputs(300, 256, 3000, seed=62))
    out_a = torch.empty(300, 256, dtype=torch.float32, device="cuda")
    T.topk_ffn_fwd_noalloc(*a, out_a, 200)
    T.topk_check()
    assert torch.equal(out_a, _reference(*a, 200))
    b = _dev(*W.ffn_inputs(129, 64, 1500, seed=63))
    out_b = torch.empty(129, 64, dtype=torch.float32, device="cuda")
    T.topk_ffn_fwd_noalloc(*b, out_b, 7)
    T.topk_check()
    assert torch.equal(out_b, _reference(*b, 7))


def test_noalloc_takes_no_device_memory():
    x, w1, w2 = _dev(*W.ffn_inputs(256, 128, 8192, seed=65))
    out = torch.empty(256, 128, dtype=torch.float32, device="cuda")
    T.topk_ffn_fwd_noalloc(x, w1, w2, out, 32)  # first call: module and symbol set-up
    T.topk_check()
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(3):
        T.topk_ffn_fwd_noalloc(x, w1, w2, out, 32)
    T.topk_check()
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0


def test_noalloc_rejects_problems_beyond_its_buffer():
    x, w1, w2 = _dev(*W.ffn_inputs(4096, 64, 65536, seed=64))
    assert T.topk_ffn_workspace_bytes(4096, 64, 65536, 512) > T.TOPK_FFN_NOALLOC_SCRATCH_BYTES
    out = torch.full((4096, 64), 7.0, dtype=torch.float32, device="cuda")
    with pytest.raises(T.TopkError) as e:
        T.topk_ffn_fwd_noalloc(x, w1, w2, out, 512)
    assert e.value.code == -7
    assert (out == 7.0).all()  # rejected before anything was launched
