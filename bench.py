#!/usr/bin/env python3
"""Throughput of top-k attention (arXiv 2106.06899, Eq. 4) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--workload NAME]

One step is one call of the whole fused path (score GEMM, top-k selection,
softmax over the k kept scores, value gather) over the full workload, inputs
resident in device memory.  Default workload: B=1, H=12, L=65536, d=64,
k=64, chunk 1024 (the long-sequence configuration).  Rank 0 prints one JSON
line.  With N > 1 (torchrun, one rank per GPU) every rank runs an
independent replica of the workload: the path has no exchange step, so there
is no collective on the data path ("replicas only", weak scaling).

--impl reference times the CPU oracle (fp64, all host cores) on bounded
samples of the same workload: the only other implementation there is.

--pass bwd times the backward pass for the cached kept set instead (Sec. 2.2):
the gradients of q, k, v (x, W1, W2) from dout and the forward pass's cache,
and the training step forward-with-cache + backward.
"""
from __future__ import annotations

import argparse
import csv
import io
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "top-k attn tokens/s and QK^T TFLOP/s (% of bf16 peak) at L=65536, k=64"
L2_BYTES = 129 * 1024 * 1024


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="long_65k")
    p.add_argument("--L", type=int, default=0, help="override Lq = Lk (profiling on a small case)")
    p.add_argument("--ffn-tokens", type=int, default=0, help="override the FF token count N (profiling)")
    p.add_argument("--e2e-steps", type=int, default=3)
    p.add_argument("--cpu-seconds", type=float, default=12.0, help="CPU work budget of the oracle baseline")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-clocks", action="store_true")
    p.add_argument("--pass", dest="which", choices=["fwd", "bwd", "plain", "decoder"], default="fwd",
                   help="bwd: time the backward pass (Sec. 2.2) for the forward pass's cache instead; "
                        "plain: the comparison path without top-k (Eq. 1 attention / the dense FF layer)")
    p.add_argument("--ffn-chunk", type=int, default=16384, help="d_ff slice of the dense FF comparison path")
    p.add_argument("--kernel-only", action="store_true",
                   help="time the device call only: no end-to-end leg, clocks or CPU baseline (profiling)")
    a = p.parse_args()
    if a.kernel_only:
        a.no_clocks, a.no_cpu_baseline, a.e2e_steps = True, True, 0
    return a


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            m = json.load(f)
        return {"hbm_gbs": m["hbm_gbs"], "bf16": m["bf16_tflops"], "bf16_sustained": m["bf16_tflops_sustained"],
                "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "source": "fallback"}


ATTN_SOURCES = ("paper_2106_06899_gb300/csrc/attn_tc.cu", "paper_2106_06899_gb300/csrc/select.cuh",
                "paper_2106_06899_gb300/csrc/common.cuh")


def profiled_traffic(w):
    """DRAM bytes per launch of the dominant kernel from the committed ncu summary, or None.

    The summary records a hash of the kernel's sources; once they have changed the counters no
    longer describe the kernel and None is returned.
    """
    import hashlib

    if w.kind != "attn" or w.name != "long_65k" or (w.Lq, w.Lk) != (65536, 65536):
        return None
    path = os.path.join(ROOT, "profiles", "attn_tc_kernel_long_65k.md")
    try:
        text = open(path).read()
        h = hashlib.sha256()
        for f in ATTN_SOURCES:
            with open(os.path.join(ROOT, f), "rb") as fh:
                h.update(fh.read())
        fields = dict(line.split(": ", 1) for line in text.splitlines() if ": " in line and line[:1].isalpha())
        if fields.get("attention_source_sha256_16") != h.hexdigest()[:16]:
            return None
        return float(fields["traffic_bytes_per_launch"])
    except (OSError, KeyError, ValueError):
        return None


def workload(args):
    from paper_2106_06899_gb300 import workloads as W

    w = W.WORKLOADS[args.workload]
    if args.L:
        w = w.with_(Lq=args.L, Lk=args.L) if w.kind == "attn" else w.with_(d_ff=args.L)
    if args.ffn_tokens and w.kind == "ffn":
        w = w.with_(N=args.ffn_tokens)
    return w


def valid_pairs(w) -> float | None:
    """(query, key) pairs that Eq. 2's masks leave valid, over all heads; None without masks."""
    if not (w.causal or w.kv_len or w.mask_p):
        return None
    import numpy as np

    from paper_2106_06899_gb300 import workloads as W

    kv, mask = W.mask_inputs(w)
    i = np.arange(w.Lq)
    lim = np.minimum(i + 1 + (w.Lk - w.Lq), w.Lk) if w.causal else np.full(w.Lq, w.Lk)
    total = 0.0
    for b in range(w.B):
        lb = np.minimum(lim, int(kv[b])) if kv is not None else lim
        if mask is None:
            total += float(lb.sum())
        else:
            m = mask[b, 0].numpy() & (np.arange(w.Lk)[None, :] < lb[:, None])
            total += float(m.sum())
    return total * w.H


def work_flops(w) -> float:
    """Algorithmic score-GEMM FLOPs of one call (every score is computed, Sec. 5); under a mask only
    the valid pairs count."""
    if w.kind == "ffn":
        return 2.0 * w.N * w.d_ff * w.d_model
    pairs = valid_pairs(w)
    if pairs is not None:
        return 2.0 * pairs * w.d
    if w.causal:  # only unmasked pairs j <= i
        pairs = w.Lq * (w.Lq + 1) / 2
        return 2.0 * w.B * w.H * pairs * w.d
    return 2.0 * w.B * w.H * w.Lq * w.Lk * w.d


# the largest k of the bf16 tensor-core attention kernels (kTcMaxK of the library)
TC_MAX_K = 512

# fp32 FMA rate of the CUDA cores: 152 SMs x 128 fp32 lanes x 2 FLOP x 2.07 GHz (maximum SM clock)
FP32_FMA_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12


def roofline(w, achieved, pk):
    """Roofline of the dominant kernel: the tcgen05 kernels against the measured bf16 tensor peak; the
    SIMT kernel (fp32 inputs, a bit mask, or k above the tensor path's 512) against the fp32 FMA rate."""
    simt = w.kind == "attn" and (w.dtype == "f32" or w.topk > TC_MAX_K or w.mask_p > 0)
    if simt:
        return {"bound": "alu", "achieved": achieved, "peak": FP32_FMA_TFLOPS, "unit": "TFLOP/s",
                "frac": achieved / FP32_FMA_TFLOPS, "traffic": None,
                "peak_source": "fp32 FMA: 152 SMs x 128 lanes x 2 FLOP x 2.07 GHz", "kernel": "attn_simt_kernel"}
    return {"bound": "tensor", "achieved": achieved, "peak": pk["bf16"], "unit": "TFLOP/s",
            "frac": achieved / pk["bf16"], "traffic": profiled_traffic(w),
            "peak_source": f"{pk['source']} bf16 dense (burst)",
            "kernel": "attn_tc_kernel" if w.kind == "attn" else "ffn kernels"}


def config_dict(w, l2_note):
    if w.kind == "ffn":
        c = {"workload": w.name, "N": w.N, "d_model": w.d_model, "d_ff": w.d_ff, "topk": w.topk}
    else:
        c = {"workload": w.name, "B": w.B, "H": w.H, "Lq": w.Lq, "Lk": w.Lk, "d": w.d, "topk": w.topk,
             "chunk": w.chunk, "causal": w.causal, "dist": w.dist}
    c["l2"] = l2_note
    c["parallelism"] = "replicas"
    return c


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for r in csv.reader(io.StringIO(out)):
            r = [x.strip() for x in r]
            if len(r) < 10:
                continue
            if self.uuid and self.uuid not in r[1]:
                continue
            rows.append(r)
        if not rows:
            return None
        sm = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        mx = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[6 + i].lower() == "active"})
        load = [s for s in sm if mx and s > 0.3 * max(mx)] or sm
        return {"sm_mhz": statistics.median(load) if load else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# ------------------------------------------------------------------ oracle timing
def oracle_masks(w):
    """Eq. 2's masks of a workload in the oracle's form (numpy), or Nones."""
    from paper_2106_06899_gb300 import workloads as W

    kv, mask = W.mask_inputs(w)
    return (None if kv is None else kv.numpy()), (None if mask is None else mask.numpy())


def oracle_rate(w, seconds: float, inputs, seed_rows: int = 0):
    """Oracle tokens/s on a bounded sample of rows of the workload (same inputs, all host cores).

    Returns (the cpu_baseline entry, the sampled rows, the oracle's result on them)."""
    import oracle
    from paper_2106_06899_gb300 import workloads as W

    cores = oracle.hardware_threads()

    def run(nrows):
        rows = W.sample_rows(w.rows, nrows, seed=seed_rows).numpy()
        t0 = time.perf_counter()
        if w.kind == "ffn":
            res = oracle.ffn(*inputs, w.topk, rows=rows)
        else:
            kv, mask = oracle_masks(w)
            res = oracle.topk_attention(*inputs, w.topk, causal=w.causal, rows=rows, kv_len=kv, mask=mask)
        return rows, res, time.perf_counter() - t0

    rows, res, t = run(max(cores, 16))
    target = max(int(len(rows) * seconds / max(t, 1e-3)), cores)
    rows, res, t = run(min(target, w.rows))
    n = len(rows)
    per_token = w.H if w.kind == "attn" else 1
    entry = {"value": (n / per_token) / t, "unit": "tokens/s", "cores": cores, "kind": "oracle",
             "sample": f"{n} of {w.rows} query rows (seeded sample), fp64 oracle, {t:.1f} s"}
    return entry, rows, res


def parity_check(w, host, dev, out, rows, ref):
    """The timed call's output on the oracle's sampled rows, under the parity rules of the tests
    (oracle/parity.py): exact index sets outside near ties, every kept key valid, outputs within
    tolerance.  The kept indices come from one extra call with index output, after the timed region
    (selection is deterministic)."""
    import torch

    import oracle
    from oracle.parity import check_rows
    from paper_2106_06899_gb300 import topk as T
    from paper_2106_06899_gb300 import workloads as W

    if w.kind == "ffn":
        _, idx, score = T.ffn(dev[0], dev[1], dev[2], w.topk, return_indices=True)
        q, k, v = (t[None, None] for t in host)
        act, dtype, d = oracle.RELU, "bf16", w.d_model
    else:
        kv, mask = W.mask_inputs(w)
        _, idx, score = T.attention(dev[0], dev[1], dev[2], w.topk, w.chunk, w.causal, return_indices=True,
                                    kv_len=None if kv is None else kv.cuda(),
                                    mask=None if mask is None else mask.cuda())
        q, k, v = host
        act, dtype, d = oracle.SOFTMAX, w.dtype, w.d
    T.topk_check()
    r = torch.as_tensor(rows, dtype=torch.long, device=out.device)
    gout = out.reshape(-1, d)[r].float().cpu().numpy()
    gidx = idx.reshape(-1, w.topk)[r].cpu().numpy()
    gscore = score.reshape(-1, w.topk)[r].cpu().numpy()
    del idx, score
    try:
        okv, omask = oracle_masks(w) if w.kind == "attn" else (None, None)
        st = check_rows(q=q, k=k, v=v, rows=rows, gpu_out=gout, gpu_idx=gidx, gpu_score=gscore, topk=w.topk,
                        dtype=dtype, act=act, causal=w.causal, ref=ref, kv_len=okv, mask=omask)
        return {"ok": True, **st}
    except AssertionError as e:
        return {"ok": False, "rows": len(rows), "error": str(e)}


# ------------------------------------------------------------------ reference arm
def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = workload(args)
    import oracle
    from paper_2106_06899_gb300 import workloads as W

    inputs = W.make_inputs(w)
    cores = oracle.hardware_threads()
    per_token = w.H if w.kind == "attn" else 1

    def step(nrows, seed):
        rows = W.sample_rows(w.rows, nrows, seed=seed).numpy()
        t0 = time.perf_counter()
        if w.kind == "ffn":
            oracle.ffn(*inputs, w.topk, rows=rows)
        else:
            kv, mask = oracle_masks(w)
            oracle.topk_attention(*inputs, w.topk, causal=w.causal, rows=rows, kv_len=kv, mask=mask)
        return len(rows), time.perf_counter() - t0

    n, t = step(max(cores, 16), 0)
    nrows = max(min(int(n * 2.0 / max(t, 1e-3)), w.rows), cores)  # about 2 s per step
    for i in range(args.warmup):
        step(nrows, 100 + i)
    times = []
    for i in range(args.steps):
        n, t = step(nrows, 1000 + i)
        times.append(t)
    tt = sum(times)
    value = (nrows * args.steps / per_token) / tt
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * tt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": config_dict(w, "host memory (CPU oracle)"),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": f"{nrows} seeded query rows of {w.rows} per step"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ replicas
def replica_throughput(ms_local: float, tokens_per_rank: int, device: str = "cuda"):
    """Whole-job throughput of independent replicas, one per rank.

    The path has no exchange step, so ranks run the same workload on their own GPU with no
    collective on the data path; the job's rate is every rank's tokens over the SLOWEST rank's
    time (MAX over ranks, the only collective, used for timing).  Returns (tokens/s, max ms).
    """
    import torch
    import torch.distributed as dist

    world = dist.get_world_size() if dist.is_available() and dist.is_initialized() else 1
    t = torch.tensor([float(ms_local)], dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    ms_max = float(t.item())
    return world * tokens_per_rank / (ms_max / 1e3), ms_max


# ------------------------------------------------------------------ our arm
def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_2106_06899_gb300 import topk as T
    from paper_2106_06899_gb300 import workloads as W

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    def barrier():
        if world > 1:
            dist.barrier()

    w = workload(args)
    host = W.make_inputs(w.with_(seed=w.seed + rank))
    dev = [t.cuda() for t in host]
    in_bytes = sum(t.numel() * t.element_size() for t in host)
    masked = False
    if w.kind == "ffn":
        out = torch.empty(w.N, w.d_model, dtype=torch.float32, device="cuda")

        def step():
            T.topk_ffn_fwd(dev[0], dev[1], dev[2], out, w.topk)
    else:
        out = torch.empty_like(dev[0])

        kv, mask = W.mask_inputs(w)
        masked = kv is not None or mask is not None
        dkv = None if kv is None else kv.cuda()
        words, mbs, mhs = T.pack_mask(mask.cuda()) if mask is not None else (None, 0, 0)

        def step():
            if masked:
                T.topk_attn_fwd_masked(dev[0], dev[1], dev[2], out, w.topk, w.chunk, w.causal, dkv, words, mbs,
                                       mhs)
            else:
                T.topk_attn_fwd(dev[0], dev[1], dev[2], out, w.topk, w.chunk, w.causal)

    flush = None
    if in_bytes <= 2 * L2_BYTES:
        flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")
        l2_note = "L2 flushed between steps (write of 2x L2 size), flush excluded by events"
    else:
        l2_note = f"inputs larger than L2 ({in_bytes / 2**20:.0f} MiB resident)"

    for _ in range(args.warmup):
        step()
    T.topk_check()
    launches_per_step = T.topk_last_launch_count()

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
    except Exception:
        pass
    sampler = ClockSampler(uuid)
    if not args.no_clocks:
        sampler.start()
        time.sleep(0.3)
    stream = torch.cuda.current_stream()
    barrier()
    torch.cuda.synchronize()
    if flush is None:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / args.steps
    else:
        tot = 0.0
        for _ in range(args.steps):
            flush.fill_(1.0)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            step()
            e1.record(stream)
            torch.cuda.synchronize()
            tot += e0.elapsed_time(e1)
        ms = tot / args.steps
    barrier()
    clocks = None if args.no_clocks else sampler.stop()
    T.topk_check()

    value, ms_max = replica_throughput(ms, w.tokens)

    # end to end through the host-buffer C-ABI entry: H2D copies, call, D2H copy, every step
    e2e = None
    if args.e2e_steps > 0:
        pinned = [t.pin_memory() for t in host]
        hout = torch.empty(out.shape, dtype=out.dtype).pin_memory()
        if w.kind == "ffn":
            def e2e_step():
                T.topk_ffn_fwd_host(pinned[0], pinned[1], pinned[2], hout, w.topk)
        elif masked:
            # no host-buffer entry takes masks: the inputs are copied on the stream, then the masked call
            # and the copy back, all through the public binding
            hkv = None if kv is None else kv.pin_memory()
            hmask = None if words is None else words.cpu().pin_memory()

            def e2e_step():
                dq_, dk_, dv_ = (t.to("cuda", non_blocking=True) for t in pinned)
                dkv_ = None if hkv is None else hkv.to("cuda", non_blocking=True)
                dm_ = None if hmask is None else hmask.to("cuda", non_blocking=True)
                T.topk_attn_fwd_masked(dq_, dk_, dv_, out, w.topk, w.chunk, w.causal, dkv_, dm_, mbs, mhs)
                hout.copy_(out, non_blocking=True)
                torch.cuda.synchronize()

            in_bytes += (0 if hkv is None else hkv.numel() * 4) + (0 if hmask is None else hmask.numel() * 4)
        else:
            def e2e_step():
                T.topk_attn_fwd_host(pinned[0], pinned[1], pinned[2], hout, w.topk, w.chunk, w.causal)
        e2e_step()
        barrier()
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            e2e_step()
        e2e_s = (time.perf_counter() - t0) / args.e2e_steps
        e2e_value, _ = replica_throughput(e2e_s * 1e3, w.tokens)
        e2e = {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": in_bytes,
               "d2h_bytes_per_step": out.numel() * out.element_size()}

    pk = peaks()
    flops = work_flops(w)
    achieved = flops / (ms_max / 1e3) / 1e12
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if w.dtype == "bf16" else "f32", "data": "synthetic",
        "config": config_dict(w, l2_note),
        "tflops": achieved,
        "roofline": roofline(w, achieved, pk),
        "e2e": e2e,
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clocks,
    }
    parity_ok = True
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"], rows, ref = oracle_rate(w, args.cpu_seconds, host)
        line["parity"] = parity_check(w, host, dev, out, rows, ref)
        parity_ok = line["parity"]["ok"]
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    if not parity_ok:
        sys.exit("parity check of the timed output failed: " + line["parity"]["error"])


# ------------------------------------------------------------------ backward pass
BWD_METRIC = "top-k backward (cached kept set, Sec. 2.2) tokens/s"


def bwd_bytes(w):
    """Compulsory HBM bytes of one backward call: the inputs q, k, v, dout and the cache (idx, score)
    read once, the fp32 gradients dq, dk, dv written once.  The gathered rows (k value and k key rows
    per query row, k query and dout rows per kept entry) come mostly from L2 and are not counted."""
    if w.kind == "ffn":
        R, Lk, d, eb = w.N, w.d_ff, w.d_model, 2
        return R * d * eb + 2 * Lk * d * eb + R * d * 4 + R * w.topk * 8 + (R * d + 2 * Lk * d) * 4
    eb = 2 if w.dtype == "bf16" else 4
    R, Lk = w.B * w.H * w.Lq, w.B * w.H * w.Lk
    return (R + 2 * Lk + R) * w.d * eb + R * w.topk * 8 + (R + 2 * Lk) * w.d * 4


def bwd_cpu_rate(w, host, dout, seconds):
    """The oracle's backward pass on a bounded head slice (all host cores): tokens/s.  Its cache is a
    random kept set (the backward pass is defined for any), not the CUDA forward pass's."""
    import oracle
    from paper_2106_06899_gb300 import workloads as W

    cores = oracle.hardware_threads()
    if w.kind == "ffn":
        n = max(16, min(w.N, int(seconds * 40)))
        idx = W.kept_sets(1, n, w.d_ff, w.topk, seed=7)
        t0 = time.perf_counter()
        oracle.ffn_bwd(host[0][:n], host[1], host[2], dout[:n].cpu(), idx.numpy())
        t = time.perf_counter() - t0
        return {"value": n / t, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                "sample": f"{n} of {w.N} tokens, random kept sets, fp64 oracle backward, {t:.1f} s"}
    h = 1
    q, k, v = (x[:, :h] for x in host)
    idx = W.kept_sets(w.B * h, w.Lq, w.Lk, w.topk, seed=7)
    t0 = time.perf_counter()
    oracle.topk_attention_bwd(q.contiguous(), k.contiguous(), v.contiguous(), dout[:, :h].cpu().contiguous(),
                              idx.numpy())
    t = time.perf_counter() - t0
    tokens = w.B * w.Lq * h / w.H
    return {"value": tokens / t, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{h} of {w.H} heads (all rows), random kept sets, fp64 oracle backward, {t:.1f} s"}


def run_backward(args):
    """Times the backward pass for the CUDA forward pass's own cache (one forward call with index
    output before timing), and the training step forward-with-cache + backward."""
    import torch

    from paper_2106_06899_gb300 import topk as T
    from paper_2106_06899_gb300 import workloads as W

    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    w = workload(args)
    host = W.make_inputs(w)
    dev = [t.cuda() for t in host]
    if w.kind == "ffn":
        dout = W.grad_output((w.N, w.d_model), dtype="f32", seed=w.seed + 1).cuda()
        out, idx, score = T.ffn(dev[0], dev[1], dev[2], w.topk, return_indices=True)
        grads = [torch.empty(t.shape, dtype=torch.float32, device="cuda") for t in dev]

        def bwd():
            T.topk_ffn_bwd(dev[0], dev[1], dev[2], dout, idx, score, *grads)

        def fwd():
            T.topk_ffn_fwd_indices(dev[0], dev[1], dev[2], out, w.topk, idx, score)
    else:
        dout = W.grad_output((w.B, w.H, w.Lq, w.d), dtype=w.dtype, seed=w.seed + 1).cuda()
        out, idx, score = T.attention(dev[0], dev[1], dev[2], w.topk, w.chunk, w.causal, return_indices=True)
        grads = [torch.empty(t.shape, dtype=torch.float32, device="cuda") for t in dev]

        def bwd():
            T.topk_attn_bwd(dev[0], dev[1], dev[2], dout, idx, score, *grads)

        def fwd():
            T.topk_attn_fwd_indices(dev[0], dev[1], dev[2], out, w.topk, w.chunk, w.causal, idx, score)
    T.topk_check()
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()

    def timed(fn):
        for _ in range(args.warmup):
            fn()
        torch.cuda.synchronize()
        tot = 0.0
        for _ in range(args.steps):
            flush.fill_(1.0)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            torch.cuda.synchronize()
            tot += e0.elapsed_time(e1)
        T.topk_check()
        return tot / args.steps

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(0).uuid)
    except Exception:
        pass
    sampler = ClockSampler(uuid)
    if not args.no_clocks:
        sampler.start()
        time.sleep(0.3)
    ms_bwd = timed(bwd)
    launches = T.topk_last_launch_count()
    ms_fwd = timed(fwd)

    def train_step():
        fwd()
        bwd()

    ms_train = timed(train_step)
    clocks = None if args.no_clocks else sampler.stop()
    pk = peaks()
    nbytes = bwd_bytes(w)
    achieved = nbytes / (ms_bwd / 1e3) / 1e9
    line = {
        "metric": BWD_METRIC, "value": w.tokens / (ms_bwd / 1e3), "unit": "tokens/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_bwd, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if w.dtype == "bf16" else "f32",
        "data": "synthetic", "config": config_dict(w, "L2 flushed between steps (write of 2x L2 size)"),
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
                     "frac": achieved / pk["hbm_gbs"], "traffic": None, "bytes_per_call": nbytes,
                     "peak_source": f"{pk['source']} HBM copy bandwidth", "kernel": "backward kernels"},
        "forward_with_cache_ms": ms_fwd,
        "train_step_ms": ms_train,
        "train_step_tokens_per_s": w.tokens / (ms_train / 1e3),
        "gpu_launches": launches * args.steps,
        "clocks": clocks,
        "e2e": None,
    }
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = bwd_cpu_rate(w, host, dout, args.cpu_seconds)
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ comparison path
PLAIN_METRIC = "plain attention / dense FF tokens/s (comparison path, no top-k)"


def run_plain(args):
    """Times the path top-k is compared with (Sec. 3): plain attention over every valid key (Eq. 1)
    or the dense FF layer (Eq. 3 without top-k), on the same workload, with the oracle's parity check
    on sampled rows after the timed region."""
    import numpy as np
    import torch

    import oracle
    from paper_2106_06899_gb300 import topk as T
    from paper_2106_06899_gb300 import workloads as W

    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    w = workload(args)
    host = W.make_inputs(w)
    dev = [t.cuda() for t in host]
    if w.kind == "ffn":
        out = torch.empty(w.N, w.d_model, dtype=torch.float32, device="cuda")

        def step():
            T.topk_vanilla_ffn_fwd(dev[0], dev[1], dev[2], out, args.ffn_chunk)

        flops = 4.0 * w.N * w.d_ff * w.d_model
        kernel = "cuBLAS GEMMs + relu_bf16_kernel"
    else:
        kv, _ = W.mask_inputs(w)
        dkv = None if kv is None else kv.cuda()
        out = torch.empty_like(dev[0])

        def step():
            T.topk_vanilla_attn_fwd(dev[0], dev[1], dev[2], out, w.chunk, w.causal, dkv)

        pairs = valid_pairs(w.with_(mask_p=0.0))
        flops = 4.0 * w.d * (pairs if pairs is not None else w.B * w.H * w.Lq * w.Lk)
        kernel = "attn_plain_kernel"
    flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        step()
    T.topk_check()
    launches = T.topk_last_launch_count()
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(0).uuid)
    except Exception:
        pass
    sampler = ClockSampler(uuid)
    if not args.no_clocks:
        sampler.start()
        time.sleep(0.3)
    torch.cuda.synchronize()
    tot = 0.0
    for _ in range(args.steps):
        flush.fill_(1.0)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step()
        e1.record(stream)
        torch.cuda.synchronize()
        tot += e0.elapsed_time(e1)
    ms = tot / args.steps
    clocks = None if args.no_clocks else sampler.stop()
    T.topk_check()
    pk = peaks()
    achieved = flops / (ms / 1e3) / 1e12
    line = {
        "metric": PLAIN_METRIC, "value": w.tokens / (ms / 1e3), "unit": "tokens/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {**config_dict(w, "L2 flushed between steps (write of 2x L2 size)"),
                   **({"ffn_chunk": args.ffn_chunk} if w.kind == "ffn" else {})},
        "tflops": achieved,
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": pk["bf16"], "unit": "TFLOP/s",
                     "frac": achieved / pk["bf16"], "traffic": None,
                     "peak_source": f"{pk['source']} bf16 dense (burst)", "kernel": kernel,
                     "flops": "4 d per valid (query, key) pair: S = QK^T and O = PV" if w.kind == "attn"
                     else "4 d_model per (token, key): both GEMMs"},
        "gpu_launches": launches * args.steps, "clocks": clocks, "e2e": None,
    }
    # parity on sampled rows against the oracle's plain attention / dense FF
    rows = W.sample_rows(w.rows, 256, seed=3).numpy()
    t0 = time.perf_counter()
    if w.kind == "ffn":
        ref = oracle.ffn_dense(*host, rows=rows)
        t = time.perf_counter() - t0
        got = out.cpu().numpy()[rows]
        # H = ReLU(x W1^T) is rounded to bf16 (relative error at most 2^-8) before the second
        # product: an element may be off by 2^-8 sum_j H_j |W2_j| (the dense layer on |W2|) plus
        # the fp32 sums
        bound = 2.0 ** -8 * oracle.ffn_dense(host[0], host[1], host[2].abs(), rows=rows) + 1e-5
    else:
        okv, _ = oracle_masks(w.with_(mask_p=0.0))
        ref = oracle.vanilla(*host, causal=w.causal, rows=rows, kv_len=okv)
        t = time.perf_counter() - t0
        got = out.float().reshape(-1, w.d).cpu().numpy()[rows]
        bound = np.full(got.shape, 2e-2)
    err = float(np.abs(got - ref).max())
    line["parity"] = {"ok": bool(np.all(np.abs(got - ref) <= bound)), "rows": len(rows), "max_err": err}
    per_token = w.H if w.kind == "attn" else 1
    line["cpu_baseline"] = {"value": len(rows) / per_token / t, "unit": "tokens/s", "cores": oracle.hardware_threads(),
                            "kind": "oracle", "sample": f"{len(rows)} of {w.rows} rows, fp64 oracle, {t:.1f} s"}
    print(json.dumps(line), flush=True)
    if not line["parity"]["ok"]:
        sys.exit(f"parity check of the plain path failed: max error {err}")


# ------------------------------------------------------------------ decoder composition
DECODER_METRIC = "12-layer decoder training step tokens/s (top-k attention, Sec. 3)"


def run_decoder(args):
    """Forward + backward of the 12-layer decoder (d_model 768, 12 heads, d_ff 3072, top-64 causal
    attention, dense FF) over one sequence of L tokens (--L, default 32768): time per step and peak
    device memory (PyTorch's allocator plus the library's pool)."""
    import torch

    from paper_2106_06899_gb300 import topk as T
    from paper_2106_06899_gb300.decoder import Decoder

    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    L = args.L or 32768
    torch.manual_seed(0)
    results = {}
    for name, topk in (("top64", 64), ("plain_sdpa", None)):
        model = Decoder(12, 768, 12, 3072, topk=topk, ffn_topk=None)
        x = torch.randn(1, L, 768, device="cuda", dtype=torch.bfloat16)

        def step():
            for p in model.parameters():
                p.grad = None
            model(x).float().pow(2).mean().backward()

        try:
            for _ in range(max(args.warmup, 1)):
                step()
            torch.cuda.synchronize()
            torch.cuda.reset_peak_memory_stats()
            T.topk_pool_usage(reset_high=True)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(args.steps):
                step()
            e1.record()
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1) / args.steps
            pool_hi, _ = T.topk_pool_usage()
            results[name] = {"ms_per_step": ms, "tokens_per_s": L / (ms / 1e3),
                             "peak_torch_bytes": torch.cuda.max_memory_allocated(), "peak_library_pool_bytes": pool_hi}
        except torch.OutOfMemoryError:
            results[name] = {"error": "out of device memory"}
        del model, x
        torch.cuda.empty_cache()
    top = results["top64"]
    line = {"metric": DECODER_METRIC, "value": top.get("tokens_per_s"), "unit": "tokens/s", "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": top.get("ms_per_step"),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": "decoder", "layers": 12, "d_model": 768, "heads": 12, "d_ff": 3072, "L": L,
                       "topk": 64, "ffn": "dense", "attention_backward": "cached kept set (Sec. 2.2)"},
            "runs": results, "e2e": None}
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    elif args.which == "bwd":
        run_backward(args)
    elif args.which == "plain":
        run_plain(args)
    elif args.which == "decoder":
        run_decoder(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
