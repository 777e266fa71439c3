"""Host logic of bench.py, CPU only: the work it counts and the roofline it reports.

* valid_pairs (the (query, key) pairs Eq. 2's masks leave valid, over all heads) against a brute-force
  count of the oracle's own mask rule (key_valid: causal bottom-right, key counts, bit mask), built
  element by element on small shapes;
* work_flops: 2 d per valid pair, the full B H Lq Lk product without masks, d_model d_ff per FF token;
* roofline: which kernel and which peak a workload is held against;
* profiled_traffic: the DRAM bytes of the committed ncu summary are used only while the summary's
  source hash matches the kernel sources, and only for the shape that was captured.
"""
import hashlib
import importlib.util
import os
import shutil

import numpy as np
import pytest

from paper_2106_06899_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _brute_pairs(w):
    kv, mask = W.mask_inputs(w)
    total = 0
    for b in range(w.B):
        for i in range(w.Lq):
            for j in range(w.Lk):
                ok = True
                if w.causal and j > i + w.Lk - w.Lq:
                    ok = False
                if kv is not None and j >= int(kv[b]):
                    ok = False
                if mask is not None and not bool(mask[b, 0, i, j]):
                    ok = False
                total += ok
    return total * w.H


@pytest.mark.parametrize("kw", [
    dict(causal=True),                                   # Lq = Lk
    dict(causal=True, Lq=5),                             # decode: the last 5 positions
    dict(kv_len=(40, 7, 0)),                             # key counts, one batch empty
    dict(mask_p=0.4),                                    # bit mask
    dict(causal=True, Lq=20, kv_len=(40, 25, 3), mask_p=0.7),
])
def test_valid_pairs_match_brute_force(kw):
    base = W.Workload("t", "attn", "bf16", seed=11, topk=4, B=3, H=2, Lq=kw.get("Lq", 40), Lk=40, d=16)
    w = base.with_(**{k: v for k, v in kw.items() if k != "Lq"})
    b = _bench()
    assert b.valid_pairs(w) == _brute_pairs(w)
    assert b.work_flops(w) == 2.0 * w.d * _brute_pairs(w)


def test_work_flops_without_masks():
    b = _bench()
    w = W.WORKLOADS["long_65k"]
    assert b.valid_pairs(w) is None
    assert b.work_flops(w) == 2.0 * 1 * 12 * 65536 * 65536 * 64  # 6.60e12, the headline's work
    f = W.WORKLOADS["ffn_65k"]
    assert b.work_flops(f) == 2.0 * 4096 * 65536 * 1024


def test_roofline_kernel_and_peak():
    b = _bench()
    pk = {"bf16": 1903.3, "source": "measured"}
    t = b.roofline(W.WORKLOADS["bert_base"], 10.0, pk)
    assert t["bound"] == "tensor" and t["peak"] == 1903.3 and t["kernel"] == "attn_tc_kernel"
    assert t["frac"] == pytest.approx(10.0 / 1903.3)
    # bf16 up to k = 512 runs on the tensor cores; fp32, bit masks and larger k on the CUDA cores
    assert b.roofline(W.WORKLOADS["bert_base_all_keys"], 1.0, pk)["bound"] == "tensor"
    for name in ("tiny_fp32", "bert_masked"):
        s = b.roofline(W.WORKLOADS[name], 1.0, pk)
        assert s["bound"] == "alu" and s["kernel"] == "attn_simt_kernel"
        assert s["peak"] == pytest.approx(152 * 128 * 2 * 2.07e9 / 1e12)
    assert b.roofline(W.WORKLOADS["bert_base"].with_(topk=b.TC_MAX_K + 1), 1.0, pk)["bound"] == "alu"
    assert b.roofline(W.WORKLOADS["ffn_65k"], 1.0, pk)["kernel"] == "ffn kernels"


def _fake_root(tmp_path, b, traffic, good_hash=True):
    root = tmp_path / "root"
    for f in b.ATTN_SOURCES:
        dst = root / f
        dst.parent.mkdir(parents=True, exist_ok=True)
        shutil.copy(os.path.join(ROOT, f), dst)
    h = hashlib.sha256()
    for f in b.ATTN_SOURCES:
        h.update((root / f).read_bytes())
    digest = h.hexdigest()[:16] if good_hash else "0" * 16
    (root / "profiles").mkdir()
    (root / "profiles" / "attn_tc_kernel_long_65k.md").write_text(
        f"# summary\n\ntraffic_bytes_per_launch: {traffic}\nattention_source_sha256_16: {digest}\n")
    return str(root)


def test_profiled_traffic_follows_the_source_hash(tmp_path, monkeypatch):
    b = _bench()
    w = W.WORKLOADS["long_65k"]
    monkeypatch.setattr(b, "ROOT", _fake_root(tmp_path / "a", b, 123456789))
    assert b.profiled_traffic(w) == 123456789.0
    # the captured shape only: another length or workload has no figure
    assert b.profiled_traffic(w.with_(Lq=32768, Lk=32768)) is None
    assert b.profiled_traffic(W.WORKLOADS["bert_base"]) is None
    # a summary of other sources describes another kernel
    monkeypatch.setattr(b, "ROOT", _fake_root(tmp_path / "b", b, 123456789, good_hash=False))
    assert b.profiled_traffic(w) is None


def test_committed_profile_is_well_formed():
    # the committed summary carries both fields the bench reads (whether its hash is current is a
    # property of the last capture, checked by the bench itself)
    text = open(os.path.join(ROOT, "profiles", "attn_tc_kernel_long_65k.md")).read()
    fields = dict(line.split(": ", 1) for line in text.splitlines() if ": " in line and line[:1].isalpha())
    assert int(fields["traffic_bytes_per_launch"]) > 0
    assert len(fields["attention_source_sha256_16"]) == 16
    int(fields["attention_source_sha256_16"], 16)
