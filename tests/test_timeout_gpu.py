"""Failure detection without a GPU fault: every pipeline wait in the tcgen05 kernels is
bounded.  A host switch makes the TMA producer withhold one key tile; the consumers' waits
run out after a short limit, the kernel drains its in-flight copies and MMAs, frees TMEM and
returns, and the host reads TOPK_ERR_TIMEOUT from the device error word.  The context stays
usable: a normal call right after is checked against the oracle."""
import numpy as np
import pytest

import oracle
from paper_2106_06899_gb300 import topk as T
from paper_2106_06899_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def test_withheld_stage_times_out_and_device_stays_usable():
    q, k, v = W.attention_inputs(1, 2, 256, 1024, 64, dtype="bf16", seed=70)
    dq, dk, dv = q.cuda(), k.cuda(), v.cuda()
    T.topk_check()  # start from a clean error word
    prev_limit = T.topk_set_wait_limit_us(200_000)  # 0.2 s per wait
    prev_skip = T.lib().topk_debug_skip_arrive(1)
    try:
        out = T.attention(dq, dk, dv, 16)
        with pytest.raises(T.TopkError) as e:
            T.topk_check()
        assert e.value.code == -4
    finally:
        T.lib().topk_debug_skip_arrive(prev_skip)
        T.topk_set_wait_limit_us(prev_limit)
    out, idx, _ = T.attention(dq, dk, dv, 16, return_indices=True)
    T.topk_check()
    gi = idx.cpu().reshape(-1, 16).numpy()
    ev, _ = oracle.eval_indices(q, k, v, gi)
    assert np.abs(out.float().cpu().reshape(-1, 64).numpy() - ev).max() <= 2e-2
