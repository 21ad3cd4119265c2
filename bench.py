#!/usr/bin/env python3
"""Benchmark of the KV-reuse hot path on GB300 ("Can I Buy Your KV Cache?",
arXiv 2606.13361).

Workload (the Qwen3-4B-shaped configuration the metric is quoted on):
  32 query heads, 8 KV heads, head dim 128, bf16; a document of L = 3774 tokens;
  one consumer continuing with q = 64 tokens, then 24 single-token decode steps;
  all 36 layers, each with its own cache (556 MB in total, far above the 129 MB
  L2), so every layer's keys stream from HBM.

One step is one pass of the whole path:
  prefill path (Sec. 5 Table 1 cost (a)):   per layer append(L) + prefill_attn(L)
  load (Algorithm 2 deserialize):           load_kv(artifact in HBM) + fork
  reuse path (cost (b)):                    per layer append(q) + reuse_attn(q),
                                            then 24 x per layer decode_step (fused append +
                                            reuse attention of the new token)
Each phase's kernels of one kind (all layers' appends, or all layers' attention)
are one CUDA graph; CUDA events between the graphs time every phase on the
launching stream.  Headline value: reuse-attention KV GB/s = algorithmic bytes
of all reuse-attention calls (prefix KV read once per call, suffix KV, Q, O)
over their device time.  Also reported: prefill-attention TFLOP/s and the
prefill/reuse cost ratios (attention only, q = 64 and q = 1).

--impl reference times the CPU oracle (the plain fp64 definition) on a bounded
sample of the same workload, on the host cores.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "reuse-attn KV GB/s vs HBM peak; prefill-attn TFLOPS; prefill/reuse cost ratio"
HQ, HKV, D = 32, 8, 128
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# ------------------------------------------------------------ arithmetic ----

def kv_bytes_per_key(hkv=HKV, d=D):
    return 2 * hkv * d * 2


NOMINAL_GBS, NOMINAL_TFLOPS = 7900.0, 2250.0  # GB300 nominal HBM3e bandwidth, dense bf16 tensor rate


def reuse_bytes(L, q, hq=HQ, hkv=HKV, d=D):
    """Algorithmic bytes of one reuse-attention call of q new rows of one
    consumer after a prefix of L: every key (prefix and suffix) read once, Q
    read, O written."""
    return (L + q) * kv_bytes_per_key(hkv, d) + 2 * q * hq * d * 2


def prefill_flops(L, hq=HQ, d=D):
    """4 * Hq * d flops per (row, visible key) pair, causal."""
    return 4 * hq * d * L * (L + 1) // 2


def reuse_flops(L, q, hq=HQ, d=D):
    return 4 * hq * d * sum(L + j + 1 for j in range(q))


# Per-launch DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) of the
# ncu captures summarised under profiles/, reported while the kernel sources
# still hash to the value recorded with the capture (null once they change).
NCU_TRAFFIC = {
    "prefill": {"files": ("kvr_attn.cu", "kvr_ptx.cuh", "kvr_internal.h"), "sha": "750a0e37a324c1f1",
                "bytes": 47.69e6, "source": "profiles/attn_prefill_qwen3-4b_L3774.md"},
    "decode": {"files": ("kvr_decode.cu", "kvr_ptx.cuh", "kvr_rope.cuh", "kvr_internal.h"),
               "sha": "97eedf642ae8f1f4", "bytes": 15.81e6, "source": "profiles/decode_step_qwen3-4b_L3774.md"},
    "reuse_q64": {"files": ("kvr_attn.cu", "kvr_ptx.cuh", "kvr_internal.h"), "sha": "750a0e37a324c1f1",
                  "bytes": 16.32e6, "source": "profiles/reuse_q64_qwen3-4b_L3774.md"},
}


def ncu_traffic(kind):
    import hashlib
    rec = NCU_TRAFFIC[kind]
    m = hashlib.sha256()
    try:
        for f in rec["files"]:
            with open(os.path.join(ROOT, "paper_2606_13361_gb300", "csrc", f), "rb") as fh:
                m.update(fh.read())
    except OSError:
        return None, rec["source"]
    return (rec["bytes"] if m.hexdigest()[:16] == rec["sha"] else None), rec["source"]


# The paper's measured M1 Pro figures for the L = 3774 document (Sec. 5,
# Table 1): prefill from scratch vs a reuse step (load + one continuation).
PAPER_M1_L3774 = {"C_prefill_s": 14.71, "C_reuse_s": 0.296}


def cost_model(c_prefill, c_load, ns=(1, 2, 10, 100, 1000)):
    """Sec. 4, Eqs. 1-3: per-call cost from scratch (flat C_prefill) and with KV
    reuse (C_prefill / N + C_load), the break-even reuse count
    N* = C_prefill / (C_prefill - C_load), and the saving over N calls."""
    return {"C_prefill_ms": c_prefill, "C_load_ms": c_load,
            "N_star": c_prefill / (c_prefill - c_load) if c_prefill > c_load else None,
            "per_call_ms": {str(n): {"from_scratch": c_prefill, "kv_reuse": c_prefill / n + c_load} for n in ns},
            "saving_ms_at_1000": 1000 * (c_prefill - c_load)}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            m = json.load(f)
        return {k: float(m[k]) for k in ("hbm_gbs", "bf16_tflops", "bf16_tflops_sustained")}, "measured"
    except (OSError, KeyError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def reduce_over_ranks(elapsed_ms: float, units: float):
    """Max elapsed and summed units over ranks (weak scaling: every rank runs
    its own replica of the workload)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return elapsed_ms, units
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([elapsed_ms], dtype=torch.float64, device=dev)
    u = torch.tensor([units], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), float(u.item())


# ---------------------------------------------------------------- clocks ----

class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms while running."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        pass

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for name, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------ CPU oracle ----

def cpu_oracle_sample(L, q, seed, budget_s=10.0, max_runs=None):
    """Time the oracle's reuse attention for one layer (q rows of one consumer
    after a prefix of L, all 32 heads) -- a bounded sample of the workload.
    Returns (per-run seconds list, threads)."""
    import numpy as np

    import oracle
    from paper_2606_13361_gb300 import inputs
    li = inputs.layer_inputs(seed, L + q, HQ, HKV, D)
    dec = oracle.bf16_decode
    _, _, qb, kb = oracle.qk_prep(dec(li.q_pre), dec(li.k_pre), dec(li.q_norm_w), dec(li.k_norm_w),
                                  np.arange(L + q), inputs.ROPE_THETA, inputs.RMS_EPS)
    k_all, v_all, qs = dec(kb), dec(li.v), dec(qb[L:])
    runs = []
    t_end = time.perf_counter() + budget_s
    while True:
        t0 = time.perf_counter()
        oracle.reuse(qs, L, k_all, v_all)
        runs.append(time.perf_counter() - t0)
        if max_runs is not None:
            if len(runs) >= max_runs:
                break
        elif time.perf_counter() > t_end:
            break
    return runs, oracle.num_threads()


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    runs, threads = cpu_oracle_sample(args.L, args.q, args.seed, budget_s=0.0,
                                      max_runs=args.warmup + args.steps)
    timed = runs[args.warmup:] or runs
    per = statistics.median(timed)
    gbs = reuse_bytes(args.L, args.q) / per / 1e9
    sample = (f"oracle reuse attention of one layer: {args.q} rows x {HQ} heads over "
              f"{args.L + args.q} keys (fp64), one run per step")
    line = {
        "impl": "reference", "metric": METRIC, "value": gbs, "unit": "GB/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": per * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic (numpy PCG64, seeded)",
        "config": workload_config(args),
        "cpu_baseline": {"value": gbs, "unit": "GB/s", "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": gbs, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


def workload_config(args):
    return {"workload": f"qwen3-4b attention: L={args.L} prefix, 1 consumer, q={args.q} then "
                        f"{args.decode} decode steps, {args.layers} layers",
            "layers": args.layers, "L": args.L, "q": args.q, "decode_steps": args.decode,
            "consumers": 1, "Hq": HQ, "Hkv": HKV, "head_dim": D,
            "l2": f"inputs larger than L2: {args.layers} distinct layer caches "
                  f"({args.layers * args.L * kv_bytes_per_key() / 1e6:.0f} MB)",
            "parallelism": "replicas"}


# ------------------------------------------------------------- GPU bench ----

class Workload:
    """Buffers, sequences and captured graphs of one step."""

    def __init__(self, args, kvr, torch, seed):
        self.a, self.kvr, self.torch = args, kvr, torch
        L, q, nd, NL = args.L, args.q, args.decode, args.layers
        dev = torch.device("cuda")
        total = L + q + nd
        pages = math.ceil(total / 128)
        self.desc = kvr.make_desc(NL, HQ, HKV, D, max_positions=total + 128)
        self.C = kvr.Context(self.desc, n_pages=4 * pages + 16, max_seqs=16)
        ctx = self.C.ctx
        g = torch.Generator(device=dev)
        g.manual_seed(seed)

        def randn(*shape):
            return torch.randn(shape, generator=g, device=dev, dtype=torch.float32).to(torch.bfloat16)

        def norm_w():
            return (1.0 + 0.1 * torch.randn((D,), generator=g, device=dev)).to(torch.bfloat16)

        self.wq = [norm_w() for _ in range(NL)]
        self.wk = [norm_w() for _ in range(NL)]
        self.doc = [(randn(L, HQ, D), randn(L, HKV, D), randn(L, HKV, D)) for _ in range(NL)]
        self.suf = [(randn(q, HQ, D), randn(q, HKV, D), randn(q, HKV, D)) for _ in range(NL)]
        self.dec = [[(randn(1, HQ, D), randn(1, HKV, D), randn(1, HKV, D)) for _ in range(NL)]
                    for _ in range(nd)]
        self.q_doc = [torch.empty((L, HQ, D), dtype=torch.bfloat16, device=dev) for _ in range(NL)]
        self.o_doc = torch.empty((L, HQ, D), dtype=torch.bfloat16, device=dev)
        self.q_suf = [torch.empty((q, HQ, D), dtype=torch.bfloat16, device=dev) for _ in range(NL)]
        self.o_suf = [torch.empty((q, HQ, D), dtype=torch.bfloat16, device=dev) for _ in range(NL)]
        self.q_dec = [[torch.empty((1, HQ, D), dtype=torch.bfloat16, device=dev) for _ in range(NL)]
                      for _ in range(nd)]
        self.o_dec = [[torch.empty((1, HQ, D), dtype=torch.bfloat16, device=dev) for _ in range(NL)]
                      for _ in range(nd)]
        self.art = torch.empty(kvr.kvr_artifact_bytes(self.desc, L), dtype=torch.uint8, device=dev)

        # --- warm every kernel once (one-time attribute setup stays out of capture)
        w = kvr.kvr_seq_open(ctx)
        kvr.kvr_append_kv(ctx, 0, [w], [0], [0, q], *self.suf[0], self.wq[0], self.wk[0], self.q_suf[0])
        kvr.kvr_reuse_attn(ctx, 0, [w], [0, q], self.q_suf[0], self.o_suf[0])
        kvr.kvr_reuse_attn(ctx, 0, [w], [0, 1], self.q_suf[0], self.o_suf[0])  # few-rows kernel
        kvr.kvr_decode_step(ctx, 0, [w], [0], [0, 1], *[x[:1] for x in self.suf[0]], self.wq[0], self.wk[0],
                            self.q_suf[0][:1], self.o_suf[0][:1])
        kvr.kvr_prefill_attn(ctx, 0, w, q, self.q_suf[0], self.o_suf[0], num_splits=1)
        torch.cuda.synchronize()
        kvr.kvr_seq_close(ctx, w)

        self.graphs = []  # (name, graph)
        self.launches_per_step = 0
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            X = kvr.kvr_seq_open(ctx)
            kvr.kvr_seq_reserve(ctx, [X], [L])
            torch.cuda.synchronize()
            n0 = kvr.kvr_launch_count(ctx)
            self._capture("prefill_append", lambda: [
                kvr.kvr_append_kv(ctx, l, [X], [0], [0, L], *self.doc[l], self.wq[l], self.wk[l],
                                  self.q_doc[l]) for l in range(NL)])
            self._capture("prefill_attn", lambda: [
                kvr.kvr_prefill_attn(ctx, l, X, L, self.q_doc[l], self.o_doc) for l in range(NL)])
            n1 = kvr.kvr_launch_count(ctx)
            # produce the artifact once (publisher, Algorithm 1) from the captured prefill
            for _, gr in self.graphs:
                gr.replay()
            torch.cuda.synchronize()
            kvr.kvr_seq_advance(ctx, [X], [L])
            meta = kvr.kvr_export_kv(ctx, X, self.art, True)
            torch.cuda.synchronize()
            n2 = kvr.kvr_launch_count(ctx)
            holder = {}

            def load():
                p = kvr.kvr_load_kv(ctx, meta, self.art, True)
                c = kvr.kvr_seq_fork(ctx, p)
                kvr.kvr_seq_reserve(ctx, [c], [q + nd])
                holder["p"], holder["c"] = p, c
            self._capture("load", load)
            Cs = holder["c"]
            self._capture("reuse_append", lambda: [
                kvr.kvr_append_kv(ctx, l, [Cs], [L], [0, q], *self.suf[l], self.wq[l], self.wk[l],
                                  self.q_suf[l]) for l in range(NL)])
            self._capture("reuse_attn", lambda: [
                kvr.kvr_reuse_attn(ctx, l, [Cs], [0, q], self.q_suf[l], self.o_suf[l])
                for l in range(NL)])
            kvr.kvr_seq_advance(ctx, [Cs], [q])
            for t in range(nd):
                pos = L + q + t
                # Algorithm 2's step: append the new token and attend, one launch per layer
                self._capture(f"decode_step_{t}", lambda t=t, pos=pos: [
                    kvr.kvr_decode_step(ctx, l, [Cs], [pos], [0, 1], *self.dec[t][l], self.wq[l],
                                        self.wk[l], self.q_dec[t][l], self.o_dec[t][l])
                    for l in range(NL)])
                kvr.kvr_seq_advance(ctx, [Cs], [1])
            n3 = kvr.kvr_launch_count(ctx)
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        self.launches_per_step = (n1 - n0) + (n3 - n2)
        self.X, self.P, self.Cs = X, holder["p"], Cs

    def _capture(self, name, fn):
        torch = self.torch
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=torch.cuda.current_stream(), capture_error_mode="thread_local"):
            fn()
        self.graphs.append((name, gr))

    def run_step(self, events):
        """Replay the step; events[i] recorded after graph i (events[0] before)."""
        events[0].record()
        for i, (_, gr) in enumerate(self.graphs):
            gr.replay()
            events[i + 1].record()


def phase_times(wl, evs_per_step):
    """Sum per-graph device times (ms) over the timed steps, by phase."""
    sums = {}
    for evs in evs_per_step:
        for i, (name, _) in enumerate(wl.graphs):
            ph = name.rsplit("_", 1)[0] if name.startswith("decode") else name
            sums[ph] = sums.get(ph, 0.0) + evs[i].elapsed_time(evs[i + 1])
    return sums


def _packed(torch, shapes, device, pinned=False):
    """One contiguous bf16 buffer holding tensors of the given shapes (each
    slice starts on a 16-byte boundary) and the views into it."""
    sizes = [math.prod(sh) for sh in shapes]
    offs, n = [], 0
    for z in sizes:
        offs.append(n)
        n += (z + 7) // 8 * 8
    buf = torch.empty(n, dtype=torch.bfloat16, device=device)
    if pinned:
        buf = buf.pin_memory()
    return buf, [buf[o:o + z].view(sh) for o, z, sh in zip(offs, sizes, shapes)]


def e2e_run(args, kvr, torch, wl, n_steps):
    """The consumer path through the public API, eager, with host buffers, as
    a serving loop runs it: the step's inputs (suffix and decode-token q/k/v
    rows of every layer, packed in one pinned host buffer) go host->device on
    a copy stream in two copies, the suffix rows first (the suffix phase waits
    for them) and the decode rows while the suffix phase runs; the library
    calls run as a user makes them (load, fork, per layer append + reuse,
    decode loop); the suffix outputs go back while the decode loop runs, the
    decode outputs at the end.  Few cross-stream waits: each one also stops
    the next library kernel from starting early.  The timed region runs from
    before the first copy to after the last one."""
    ctx = wl.C.ctx
    L, q, nd, NL = args.L, args.q, args.decode, args.layers
    src = [t for lay in wl.suf for t in lay] + [t for st in wl.dec for lay in st for t in lay]
    h_in, h_views = _packed(torch, [t.shape for t in src], "cpu", pinned=True)
    for h, t in zip(h_views, src):
        h.copy_(t.cpu())
    d_in, d_views = _packed(torch, [t.shape for t in src], "cuda")
    out_shapes = [(q, HQ, D)] * NL + [(1, HQ, D)] * (nd * NL)
    d_out, outs = _packed(torch, out_shapes, "cuda")
    h_out = torch.empty_like(d_out, device="cpu").pin_memory()
    qo = [torch.empty((q, HQ, D), dtype=torch.bfloat16, device="cuda") for _ in range(NL)]
    meta = kvr.kvr_artifact_meta(wl.desc.model_id, kvr.KVR_DTYPE_BF16, L)

    def span(buf, views, i0, i1):  # element range of views[i0:i1] in their packed buffer
        b0 = (views[i0].data_ptr() - buf.data_ptr()) // 2
        b1 = (views[i1 - 1].data_ptr() - buf.data_ptr()) // 2 + views[i1 - 1].numel()
        return slice(b0, b1)

    in_chunks = [span(d_in, d_views, 0, 3 * NL), span(d_in, d_views, 3 * NL, len(d_views))]
    out_chunks = [span(d_out, outs, 0, NL), span(d_out, outs, NL, len(outs))]
    main = torch.cuda.current_stream()
    cs = torch.cuda.Stream()
    times = []
    for _ in range(n_steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        cs.wait_stream(main)
        ev_in = []
        with torch.cuda.stream(cs):
            for sl in in_chunks:
                d_in[sl].copy_(h_in[sl], non_blocking=True)
                ev = torch.cuda.Event()
                ev.record(cs)
                ev_in.append(ev)

        def send_back(k):
            ev = torch.cuda.Event()
            ev.record(main)
            cs.wait_event(ev)
            with torch.cuda.stream(cs):
                h_out[out_chunks[k]].copy_(d_out[out_chunks[k]], non_blocking=True)

        p = kvr.kvr_load_kv(ctx, meta, wl.art, True)
        c = kvr.kvr_seq_fork(ctx, p)
        main.wait_event(ev_in[0])
        for l in range(NL):
            qq, kk, vv = d_views[3 * l: 3 * l + 3]
            kvr.kvr_append_kv(ctx, l, [c], [L], [0, q], qq, kk, vv, wl.wq[l], wl.wk[l], qo[l])
            kvr.kvr_reuse_attn(ctx, l, [c], [0, q], qo[l], outs[l])
        kvr.kvr_seq_advance(ctx, [c], [q])
        send_back(0)
        base = 3 * NL
        main.wait_event(ev_in[1])
        for t in range(nd):
            for l in range(NL):
                i = base + 3 * (t * NL + l)
                kvr.kvr_decode_step(ctx, l, [c], [L + q + t], [0, 1], d_views[i], d_views[i + 1], d_views[i + 2],
                                    wl.wq[l], wl.wk[l], None, outs[NL + t * NL + l])
            kvr.kvr_seq_advance(ctx, [c], [1])
        send_back(1)
        main.wait_stream(cs)
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
        kvr.kvr_seq_close(ctx, c)
        kvr.kvr_seq_close(ctx, p)
    st = kvr.kvr_sync_status(ctx)
    if st != kvr.KVR_OK:
        raise RuntimeError(f"device status {st}: {kvr.kvr_last_error()}")
    h2d = h_in.numel() * h_in.element_size()
    d2h = h_out.numel() * h_out.element_size()
    return statistics.median(times), h2d, d2h


def _time_call(torch, fn, reps):
    """Median CUDA-event time (ms) of fn() over reps calls after one warm-up;
    fn may return a cleanup callable, run outside the timed region."""
    times = []
    for _ in range(reps + 1):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        done = fn()
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
        if callable(done):
            done()
    return statistics.median(times[1:])


def run_artifact_io(kvr, torch, wl, reps=5):
    """Artifact transfer rates of Algorithms 1-2 on this GPU, bf16 and the
    Sec. 5 int8 encoding: kvr_load_kv from device memory and from pinned host
    memory (the consumer that fetched the artifact into host RAM), and the
    export to pinned host memory (the publisher storing it).  Rates are
    artifact bytes / time; int8 export also reads the bf16 cache twice (max |x|
    per tensor, then the codes)."""
    ctx = wl.C.ctx
    L = wl.a.L
    n16 = wl.art.numel()
    n8 = kvr.kvr_artifact_bytes_q8(wl.desc, L)
    meta16 = kvr.kvr_artifact_meta(wl.desc.model_id, kvr.KVR_DTYPE_BF16, L)
    meta8 = kvr.kvr_artifact_meta(wl.desc.model_id, kvr.KVR_DTYPE_Q8, L)
    host16 = wl.art.cpu().pin_memory()
    dev8 = torch.empty(n8, dtype=torch.uint8, device="cuda")
    host8 = torch.empty(n8, dtype=torch.uint8).pin_memory()
    out = {}

    def load(meta, src, on_dev):
        p = kvr.kvr_load_kv(ctx, meta, src, on_dev)
        return lambda: kvr.kvr_seq_close(ctx, p)

    cases = (
        ("bf16_load_device", n16, lambda: load(meta16, wl.art, True)),
        ("bf16_load_pinned_host", n16, lambda: load(meta16, host16, False)),
        ("bf16_export_pinned_host", n16, lambda: kvr.kvr_export_kv(ctx, wl.P, host16, False)),
        ("int8_export_device", n8, lambda: kvr.kvr_export_kv_q8(ctx, wl.P, dev8, True)),
        ("int8_export_pinned_host", n8, lambda: kvr.kvr_export_kv_q8(ctx, wl.P, host8, False)),
        ("int8_load_device", n8, lambda: load(meta8, dev8, True)),
        ("int8_load_pinned_host", n8, lambda: load(meta8, host8, False)),
    )
    for name, nbytes, fn in cases:
        ms = _time_call(torch, fn, reps)
        out[name] = {"ms": ms, "GB_s": nbytes / (ms * 1e-3) / 1e9}
    st = kvr.kvr_sync_status(ctx)
    if st != kvr.KVR_OK:
        raise RuntimeError(f"device status {st}: {kvr.kvr_last_error()}")
    out["artifact_bytes"] = {"bf16": n16, "int8": n8, "ratio": n16 / n8}
    out["note"] = (f"one artifact of the workload ({wl.a.layers} layers, L={L}); tile kernels for device and "
                   f"pinned host buffers; median of {reps}")
    return out


def run_int8_probe(kvr, torch, L=692, steps=32, vocab=4096, seed=12):
    """Sec. 5's size-vs-exactness probe on the library: one Qwen3-4B-shaped
    layer, a 692-token context stored at bf16 and at int8, then 32 greedy
    decode steps from each through kvr_decode_step and a synthetic head
    (logits = W_head . O, next token's q/k/v = row of a token table; stand-ins
    for the weights).  Reports how many greedy tokens agree with the bf16 path,
    the first step that differs, and the attention-output error of the first
    step."""
    import numpy as np
    from paper_2606_13361_gb300 import inputs
    dev = torch.device("cuda")
    desc = kvr.make_desc(1, HQ, HKV, D, max_positions=L + steps + 128)
    full = kvr.make_desc(36, HQ, HKV, D, max_positions=L + steps + 128)
    C = kvr.Context(desc, n_pages=4 * (L // 128 + 2), max_seqs=8)
    ctx = C.ctx
    li = inputs.layer_inputs(seed, L, HQ, HKV, D)
    W, E = inputs.head_tables(seed + 1, vocab, HQ, HKV, D)

    def t16(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(dev)

    Wt, Et = t16(W).float(), t16(E)
    wq, wk = t16(li.q_norm_w), t16(li.k_norm_w)
    x = kvr.kvr_seq_open(ctx)
    q_doc = torch.empty((L, HQ, D), dtype=torch.bfloat16, device=dev)
    kvr.kvr_append_kv(ctx, 0, [x], [0], [0, L], t16(li.q_pre), t16(li.k_pre), t16(li.v), wq, wk, q_doc)
    kvr.kvr_seq_advance(ctx, [x], [L])
    art16 = torch.empty(kvr.kvr_artifact_bytes(desc, L), dtype=torch.uint8, device=dev)
    art8 = torch.empty(kvr.kvr_artifact_bytes_q8(desc, L), dtype=torch.uint8, device=dev)
    m16 = kvr.kvr_export_kv(ctx, x, art16, True)
    m8 = kvr.kvr_export_kv_q8(ctx, x, art8, True)
    hq, hk = HQ * D, (HQ + HKV) * D
    toks, first_o = {}, {}
    for name, meta, art in (("bf16", m16, art16), ("int8", m8, art8)):
        c = kvr.kvr_seq_fork(ctx, kvr.kvr_load_kv(ctx, meta, art, True))
        tok, out = 0, []
        for t in range(steps):
            row = Et[tok]
            o = torch.empty((1, HQ, D), dtype=torch.bfloat16, device=dev)
            kvr.kvr_decode_step(ctx, 0, [c], [L + t], [0, 1], row[:hq].view(1, HQ, D),
                                row[hq:hk].view(1, HKV, D), row[hk:].view(1, HKV, D), wq, wk, None, o)
            kvr.kvr_seq_advance(ctx, [c], [1])
            if t == 0:
                first_o[name] = o.float()
            tok = int(torch.argmax(Wt @ o.float().reshape(-1)))
            out.append(tok)
        toks[name] = out
    st = kvr.kvr_sync_status(ctx)
    if st != kvr.KVR_OK:
        raise RuntimeError(f"device status {st}: {kvr.kvr_last_error()}")
    same = [a == b for a, b in zip(toks["bf16"], toks["int8"])]
    diff = (first_o["int8"] - first_o["bf16"]).reshape(-1)
    ref = first_o["bf16"].reshape(-1)
    C.close()
    return {"context_tokens": L, "greedy_steps": steps,
            "artifact_MB": {"bf16": kvr.kvr_artifact_bytes(full, L) / 1e6, "int8": kvr.kvr_artifact_bytes_q8(full, L) / 1e6,
                            "note": "sizes of the 36-layer artifact at this L (the probe runs one layer)"},
            "tokens_matching_bf16": int(sum(same)),
            "first_divergence_step": (same.index(False) if False in same else None),
            "step0_attention_output": {"max_abs_diff": float(diff.abs().max()),
                                       "rel_rms_diff": float(diff.norm() / ref.norm())},
            "paper_probe": "Sec. 5: 102.1 -> 51.1 MB, 16/32 greedy tokens match (Qwen3-4B, real weights)"}


def _graph(torch, fn):
    gr = torch.cuda.CUDAGraph()
    st = torch.cuda.Stream()
    st.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(st):
        with torch.cuda.graph(gr, stream=st, capture_error_mode="thread_local"):
            fn()
    torch.cuda.current_stream().wait_stream(st)
    torch.cuda.synchronize()
    return gr


def _time_graph(torch, gr, reps):
    gr.replay()
    torch.cuda.synchronize()
    times = []
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        gr.replay()
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    return statistics.median(times)


def run_sweep(kvr, torch, peaks, lengths, reps=5, q=64, seed=1, min_bytes=512 << 20):
    """L sweep (Qwen3-4B layer shapes): prefill attention over L, reuse
    attention of q rows after an L-token document, and one decode step (fused
    append + attention).  For each L the cache holds enough layers for the
    working set to exceed L2 (>= 512 MB); each call type is one CUDA graph with
    one call per layer, timed as the main workload is (per call = graph time /
    layers, median of reps replays)."""
    out = []
    for L in lengths:
        NL = int(min(128, max(2, math.ceil(min_bytes / (L * kv_bytes_per_key())))))
        desc = kvr.make_desc(NL, HQ, HKV, D, max_positions=L + q + 256)
        C = kvr.Context(desc, n_pages=2 * ((L + 127) // 128) + 8, max_seqs=8)
        ctx = C.ctx
        g = torch.Generator(device="cuda")
        g.manual_seed(seed + L)

        def rn(*shape):
            return torch.randn(shape, generator=g, device="cuda").to(torch.bfloat16)

        w = (1.0 + 0.1 * torch.randn((2, D), generator=g, device="cuda")).to(torch.bfloat16)
        pre = (rn(L, HQ, D), rn(L, HKV, D), rn(L, HKV, D))  # same pre-norm tokens for every layer
        x = kvr.kvr_seq_open(ctx)
        qx = torch.empty((L, HQ, D), dtype=torch.bfloat16, device="cuda")
        for l in range(NL):
            kvr.kvr_append_kv(ctx, l, [x], [0], [0, L], *pre, w[0], w[1], qx)
        ox = torch.empty_like(qx)
        kvr.kvr_prefill_attn(ctx, 0, x, L, qx, ox)
        t_pre = _time_graph(torch, _graph(torch, lambda: [kvr.kvr_prefill_attn(ctx, l, x, L, qx, ox)
                                                          for l in range(NL)]), reps) / NL
        kvr.kvr_seq_advance(ctx, [x], [L])
        c = kvr.kvr_seq_fork(ctx, x)
        suf = (rn(q, HQ, D), rn(q, HKV, D), rn(q, HKV, D))
        qs = torch.empty((q, HQ, D), dtype=torch.bfloat16, device="cuda")
        for l in range(NL):
            kvr.kvr_append_kv(ctx, l, [c], [L], [0, q], *suf, w[0], w[1], qs)
        os_ = torch.empty_like(qs)
        kvr.kvr_reuse_attn(ctx, 0, [c], [0, q], qs, os_)
        t_reu = _time_graph(torch, _graph(torch, lambda: [kvr.kvr_reuse_attn(ctx, l, [c], [0, q], qs, os_)
                                                          for l in range(NL)]), reps) / NL
        kvr.kvr_seq_advance(ctx, [c], [q])
        dq, dk, dv = rn(1, HQ, D), rn(1, HKV, D), rn(1, HKV, D)
        od = torch.empty((1, HQ, D), dtype=torch.bfloat16, device="cuda")
        kvr.kvr_decode_step(ctx, 0, [c], [L + q], [0, 1], dq, dk, dv, w[0], w[1], None, od)
        t_dec = _time_graph(torch, _graph(torch, lambda: [
            kvr.kvr_decode_step(ctx, l, [c], [L + q], [0, 1], dq, dk, dv, w[0], w[1], None, od)
            for l in range(NL)]), reps) / NL
        if kvr.kvr_sync_status(ctx) != kvr.KVR_OK:
            raise RuntimeError(kvr.kvr_last_error())
        pf = prefill_flops(L) / (t_pre * 1e-3) / 1e12
        rg = reuse_bytes(L, q) / (t_reu * 1e-3) / 1e9
        dg = reuse_bytes(L + q, 1) / (t_dec * 1e-3) / 1e9
        out.append({"L": L, "layers": NL, "prefill_ms": t_pre, "reuse_q64_ms": t_reu, "decode_step_ms": t_dec,
                    "prefill_tflops": pf, "prefill_frac_bf16_burst": pf / peaks["bf16_tflops"],
                    "reuse_q64_gbs": rg, "reuse_q64_frac_hbm": rg / peaks["hbm_gbs"],
                    "decode_gbs": dg, "decode_frac_hbm": dg / peaks["hbm_gbs"],
                    "ratio_q64": t_pre / t_reu, "ratio_q1": t_pre / t_dec})
        C.close()
        del qx, ox, pre
    return out


def run_q8_resident(kvr, torch, peaks, lengths=(3838, 32768), reps=5, seed=5, min_bytes=512 << 20):
    """Decode over an int8-resident prefix (Sec. 5's int8 artifact kept as codes
    in HBM, dequantised inside the decode kernel's tile load) against decode
    over the same artifact loaded as bf16 (Qwen3-4B layer shapes, one consumer,
    one new token per step).  The int8 side reads one byte per element of the
    full prefix pages (exact f16 codes in shared memory, the scales applied to
    scores and probabilities); its outputs differ from the bf16 side's only by
    the bf16 rounding of the dequantised cache.  Per L the cache holds enough
    layers for the int8 working set to exceed L2; one CUDA graph of one decode
    step per layer, per call = graph time / layers."""
    out = []
    for L in lengths:
        NL = int(min(36, max(2, math.ceil(min_bytes / (L * kv_bytes_per_key() // 2)))))
        desc = kvr.make_desc(NL, HQ, HKV, D, max_positions=L + 256)
        pages = (L + 127) // 128
        C = kvr.Context(desc, n_pages=4 * pages + 16, max_seqs=8)
        ctx = C.ctx
        g = torch.Generator(device="cuda")
        g.manual_seed(seed + L)

        def rn(*shape):
            return torch.randn(shape, generator=g, device="cuda").to(torch.bfloat16)

        w = (1.0 + 0.1 * torch.randn((2, D), generator=g, device="cuda")).to(torch.bfloat16)
        x = kvr.kvr_seq_open(ctx)
        pre = (rn(L, HQ, D), rn(L, HKV, D), rn(L, HKV, D))
        qx = torch.empty((L, HQ, D), dtype=torch.bfloat16, device="cuda")
        for l in range(NL):
            kvr.kvr_append_kv(ctx, l, [x], [0], [0, L], *pre, w[0], w[1], qx)
        kvr.kvr_seq_advance(ctx, [x], [L])
        del pre, qx
        art = torch.empty(kvr.kvr_artifact_bytes_q8(desc, L), dtype=torch.uint8, device="cuda")
        meta = kvr.kvr_export_kv_q8(ctx, x, art, True)
        kvr.kvr_seq_close(ctx, x)
        dq, dk, dv = rn(1, HQ, D), rn(1, HKV, D), rn(1, HKV, D)
        row = {"L": L, "layers": NL}
        outs = {}
        for kind, load in (("bf16", kvr.kvr_load_kv), ("int8_resident", kvr.kvr_load_kv_q8_resident)):
            p = load(ctx, meta, art, True)
            c = kvr.kvr_seq_fork(ctx, p)
            od = torch.empty((1, HQ, D), dtype=torch.bfloat16, device="cuda")
            kvr.kvr_decode_step(ctx, 0, [c], [L], [0, 1], dq, dk, dv, w[0], w[1], None, od)
            t = _time_graph(torch, _graph(torch, lambda: [
                kvr.kvr_decode_step(ctx, l, [c], [L], [0, 1], dq, dk, dv, w[0], w[1], None, od)
                for l in range(NL)]), reps) / NL
            outs[kind] = od.clone()
            full = (L // 128) * 128
            moved = reuse_bytes(L, 1) - (full * kv_bytes_per_key() // 2 if kind != "bf16" else 0)
            row[kind] = {"decode_step_ms": t, "cache_bytes_read": moved,
                         "gbs": moved / (t * 1e-3) / 1e9, "frac_hbm": moved / (t * 1e-3) / 1e9 / peaks["hbm_gbs"]}
            kvr.kvr_seq_close(ctx, c)
            kvr.kvr_seq_close(ctx, p)
        if kvr.kvr_sync_status(ctx) != kvr.KVR_OK:
            raise RuntimeError(kvr.kvr_last_error())
        row["max_abs_diff_vs_bf16"] = float((outs["bf16"].float() - outs["int8_resident"].float()).abs().max())
        row["speedup"] = row["bf16"]["decode_step_ms"] / row["int8_resident"]["decode_step_ms"]
        out.append(row)
        C.close()
        del art
    return out


def run_serving(kvr, torch, peaks, layers=36, L=3774, B=64, q=128, steps=5, seed=2):
    """Shared-prefix serving: one document, B consumers x q new tokens, one
    reuse call per layer (each prefix key tile staged once per query block and
    served to every consumer row in it).  Graph of all layers' appends, then
    all layers' reuse calls."""
    desc = kvr.make_desc(layers, HQ, HKV, D, max_positions=L + q + 256)
    pages = (L + 127) // 128 + B * ((q + 127) // 128 + 2) + 8
    C = kvr.Context(desc, n_pages=pages, max_seqs=B + 4)
    ctx = C.ctx
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    art = torch.randn(kvr.kvr_artifact_bytes(desc, L) // 2, generator=g, device="cuda").to(torch.bfloat16)
    p = kvr.kvr_load_kv(ctx, kvr.kvr_artifact_meta(desc.model_id, 1, L), art, True)
    seqs = [kvr.kvr_seq_fork(ctx, p) for _ in range(B)]
    kvr.kvr_seq_reserve(ctx, seqs, [q] * B)
    T = B * q
    qp = torch.randn((T, HQ, D), generator=g, device="cuda").to(torch.bfloat16)
    kp = torch.randn((T, HKV, D), generator=g, device="cuda").to(torch.bfloat16)
    vv = torch.randn((T, HKV, D), generator=g, device="cuda").to(torch.bfloat16)
    w = (1.0 + 0.1 * torch.randn((2, D), generator=g, device="cuda")).to(torch.bfloat16)
    qo = torch.empty_like(qp)
    oo = torch.empty_like(qp)
    cu = [b * q for b in range(B + 1)]
    kvr.kvr_reuse_attn(ctx, 0, seqs[:1], [0, q], qo, oo)  # warm
    torch.cuda.synchronize()
    graphs = [_graph(torch, lambda: [kvr.kvr_append_kv(ctx, l, seqs, [L] * B, cu, qp, kp, vv, w[0], w[1], qo)
                                     for l in range(layers)]),
              _graph(torch, lambda: [kvr.kvr_reuse_attn(ctx, l, seqs, cu, qo, oo) for l in range(layers)])]
    torch.cuda.synchronize()
    for gr in graphs:
        gr.replay()
    torch.cuda.synchronize()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for e in ev:
        e[0].record()
        graphs[0].replay()
        e[1].record()
        graphs[1].replay()
        e[2].record()
    torch.cuda.synchronize()
    if kvr.kvr_sync_status(ctx) != kvr.KVR_OK:
        raise RuntimeError(kvr.kvr_last_error())
    t_app = statistics.median(e[0].elapsed_time(e[1]) for e in ev) / layers
    t_att = statistics.median(e[1].elapsed_time(e[2]) for e in ev) / layers
    flops = B * reuse_flops(L, q)
    once = L * kv_bytes_per_key() + B * q * kv_bytes_per_key() + 2 * T * HQ * D * 2
    reread = B * (L + q) * kv_bytes_per_key() + 2 * T * HQ * D * 2
    tf = flops / (t_att * 1e-3) / 1e12
    C.close()
    return {"workload": f"{layers} layers, L={L} shared prefix, {B} consumers x q={q}",
            "reuse_ms_per_layer": t_att, "append_ms_per_layer": t_app,
            "reuse_tflops": tf, "reuse_frac_bf16_burst": tf / peaks["bf16_tflops"],
            "algorithmic_bytes_per_layer": once, "bytes_if_prefix_reread_per_consumer": reread,
            "effective_gbs_prefix_once": once / (t_att * 1e-3) / 1e9,
            "bound": "tensor (%.0f flop/B)" % (flops / once)}


QWEN_HIDDEN, QWEN_INTER = 2560, 9728
PAPER_TABLE1_L3774_SPEEDUP = 49.7


def run_layer_cost(kvr, torch, peaks, layers=36, L=3774, q=64, reps=3, seed=4):
    """Whole-model cost on GB300 (Sec. 5, Table 1 times whole Qwen3-4B
    forwards): 36 Qwen3-4B-shaped decoder layers with random weights
    (kvr_layer_forward: norms, projections, QK-norm + RoPE, attention, SwiGLU
    MLP) for prefill of the L-token document from scratch, a q-token
    continuation over the loaded artifact, and one decode token.  Each is one
    CUDA graph of the 36 layer calls; the projections are this library's
    tcgen05 GEMM (the weight-streaming GEMV for the decode token)."""
    dev = torch.device("cuda")
    H, I = QWEN_HIDDEN, QWEN_INTER
    desc = kvr.make_desc(layers, HQ, HKV, D, max_positions=L + q + 256)
    ld = kvr.kvr_layer_desc(H, I)
    C = kvr.Context(desc, n_pages=3 * ((L + q) // 128 + 4), max_seqs=8)
    ctx = C.ctx
    g = torch.Generator(device=dev)
    g.manual_seed(seed)

    def lin(o, i):
        return (torch.randn((o, i), generator=g, device=dev) / math.sqrt(i)).to(torch.bfloat16)

    def nw(n):
        return (1 + 0.1 * torch.randn((n,), generator=g, device=dev)).to(torch.bfloat16)

    Wd = [{"input_norm": nw(H), "wq": lin(HQ * D, H), "wk": lin(HKV * D, H), "wv": lin(HKV * D, H),
           "q_norm": nw(D), "k_norm": nw(D), "wo": lin(H, HQ * D), "post_norm": nw(H),
           "w_gate_up": lin(2 * I, H), "w_down": lin(H, I)} for _ in range(layers)]
    Ws = [kvr.layer_weights(w) for w in Wd]
    weight_bytes = sum(t.numel() * 2 for w in Wd for t in w.values())
    ws = torch.empty(kvr.kvr_layer_workspace_bytes(desc, ld, L), dtype=torch.uint8, device=dev)
    h_doc = torch.randn((L, H), generator=g, device=dev).to(torch.bfloat16)
    h_q = torch.randn((q, H), generator=g, device=dev).to(torch.bfloat16)
    h_t = torch.randn((1, H), generator=g, device=dev).to(torch.bfloat16)
    bufs = {T: [torch.empty((T, H), dtype=torch.bfloat16, device=dev) for _ in range(2)] for T in (L, q, 1)}

    def model(seq, start, h0):
        T = h0.shape[0]
        src = h0
        for l in range(layers):
            dst = bufs[T][l % 2]
            kvr.kvr_layer_forward(ctx, l, ld, Ws[l], [seq], [start], [0, T], src, dst, ws)
            src = dst

    x = kvr.kvr_seq_open(ctx)
    kvr.kvr_seq_reserve(ctx, [x], [L])
    model(x, 0, h_doc)  # warm: kernel attributes
    torch.cuda.synchronize()
    g_pre = _graph(torch, lambda: model(x, 0, h_doc))
    t_pre = _time_graph(torch, g_pre, reps)
    kvr.kvr_seq_advance(ctx, [x], [L])
    art = torch.empty(kvr.kvr_artifact_bytes(desc, L), dtype=torch.uint8, device=dev)
    meta = kvr.kvr_export_kv(ctx, x, art, True)
    p = kvr.kvr_load_kv(ctx, meta, art, True)
    c = kvr.kvr_seq_fork(ctx, p)
    kvr.kvr_seq_reserve(ctx, [c], [q + 1])
    model(c, L, h_q)
    torch.cuda.synchronize()
    g_q = _graph(torch, lambda: model(c, L, h_q))
    t_q = _time_graph(torch, g_q, reps)
    kvr.kvr_seq_advance(ctx, [c], [q])
    model(c, L + q, h_t)
    torch.cuda.synchronize()
    g_1 = _graph(torch, lambda: model(c, L + q, h_t))
    t_1 = _time_graph(torch, g_1, reps)
    def load():
        s_ = kvr.kvr_load_kv(ctx, meta, art, True)
        return lambda: kvr.kvr_seq_close(ctx, s_)

    t_load = _time_call(torch, load, reps)
    st = kvr.kvr_sync_status(ctx)
    if st != kvr.KVR_OK:
        raise RuntimeError(f"device status {st}: {kvr.kvr_last_error()}")
    C.close()
    f_pre = layers * oracle_free_layer_flops(L, L * (L + 1) // 2, H, I)
    f_q = layers * oracle_free_layer_flops(q, sum(L + j + 1 for j in range(q)), H, I)
    f_1 = layers * oracle_free_layer_flops(1, L + q + 1, H, I)
    kv_q = layers * reuse_bytes(L, q)
    kv_1 = layers * reuse_bytes(L + q, 1)
    return {
        "workload": f"{layers} Qwen3-4B-shaped layers (hidden {H}, MLP {I}, {HQ}/{HKV} heads x {D}), random "
                    f"weights; document L={L}, continuation q={q}, then one decode token",
        "prefill_ms": t_pre, "prefill_tflops": f_pre / (t_pre * 1e-3) / 1e12,
        "reuse_q64_ms": t_q, "reuse_q64_tflops": f_q / (t_q * 1e-3) / 1e12,
        "decode_ms": t_1,
        "decode_gbs": (weight_bytes + kv_1) / (t_1 * 1e-3) / 1e9,
        "decode_frac_hbm": (weight_bytes + kv_1) / (t_1 * 1e-3) / 1e9 / peaks["hbm_gbs"],
        "artifact_load_ms": t_load,
        "weight_bytes": weight_bytes, "kv_bytes_q64": kv_q, "kv_bytes_decode": kv_1,
        "ratio_prefill_over_reuse_q64": t_pre / t_q,
        "ratio_prefill_over_decode": t_pre / t_1,
        "ratio_prefill_over_load_plus_decode": t_pre / (t_load + t_1),
        "paper_table1_L3774_speedup": PAPER_TABLE1_L3774_SPEEDUP,
        "note": "whole-model ratio on GB300 vs the paper's M1 Pro figure (one continuation token over a resident "
                "cache); the projections are this library's tcgen05 GEMM (GEMV at one token); decode_gbs counts the "
                "36 layers' weights plus the KV read",
    }


def oracle_free_layer_flops(T, pairs, hidden, inter, hq=HQ, hkv=HKV, d=D):
    """2 x multiply-adds of one layer for T new tokens with `pairs` visible
    (row, key) pairs per head: projections, MLP, attention."""
    return 2 * T * hidden * (2 * hq * d + 2 * hkv * d) + 6 * T * hidden * inter + 4 * hq * d * pairs


def run_hotdoc(kvr, torch, peaks, layers=4, L=32768, B=256, steps=24, seed=3, reps=3):
    """Hot document: a 32K-token prefix shared by B consumers with ragged
    suffixes (uniform in [16, 512]), one batched reuse call per layer, then
    `steps` decode steps of all B consumers together (one token each, one call
    per layer).  Per-layer cost does not depend on how many layers the cache
    holds; `layers` layers (each 134 MB of prefix KV, more than L2) are timed
    and the per-layer figures stand for every layer of the 36-layer model."""
    from paper_2606_13361_gb300 import inputs
    qs = [int(x) for x in inputs.ragged_lengths(seed, B, 16, 512)]
    T = sum(qs)
    desc = kvr.make_desc(layers, HQ, HKV, D, max_positions=L + 512 + steps + 256)
    pages = (L + 127) // 128 + B * ((512 + steps + 127) // 128 + 1) + 8
    C = kvr.Context(desc, n_pages=pages, max_seqs=B + 4)
    ctx = C.ctx
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)

    def rn(*shape):
        return torch.randn(shape, generator=g, device="cuda").to(torch.bfloat16)
    art = rn(kvr.kvr_artifact_bytes(desc, L) // 2)
    p = kvr.kvr_load_kv(ctx, kvr.kvr_artifact_meta(desc.model_id, 1, L), art, True)
    del art
    seqs = [kvr.kvr_seq_fork(ctx, p) for _ in range(B)]
    kvr.kvr_seq_reserve(ctx, seqs, [q + steps for q in qs])
    qp, kp, vv = rn(T, HQ, D), rn(T, HKV, D), rn(T, HKV, D)
    w = (1.0 + 0.1 * torch.randn((2, D), generator=g, device="cuda")).to(torch.bfloat16)
    qo, oo = torch.empty_like(qp), torch.empty_like(qp)
    cu = [0]
    for q in qs:
        cu.append(cu[-1] + q)
    dec = [(rn(B, HQ, D), rn(B, HKV, D), rn(B, HKV, D)) for _ in range(steps)]
    dq, do = torch.empty((B, HQ, D), dtype=torch.bfloat16, device="cuda"), torch.empty((B, HQ, D), dtype=torch.bfloat16, device="cuda")
    cud = list(range(B + 1))
    torch.cuda.synchronize()
    graphs = [_graph(torch, lambda: [kvr.kvr_append_kv(ctx, l, seqs, [L] * B, cu, qp, kp, vv, w[0], w[1], qo)
                                     for l in range(layers)]),
              _graph(torch, lambda: [kvr.kvr_reuse_attn(ctx, l, seqs, cu, qo, oo) for l in range(layers)])]
    kvr.kvr_seq_advance(ctx, seqs, qs)
    for t in range(steps):
        graphs.append(_graph(torch, lambda t=t: [
            kvr.kvr_decode_step(ctx, l, seqs, [L + q + t for q in qs], cud, *dec[t], w[0], w[1], dq, do)
            for l in range(layers)]))
        kvr.kvr_seq_advance(ctx, seqs, [1] * B)
    for gr in graphs:
        gr.replay()
    torch.cuda.synchronize()
    times = [[] for _ in graphs]
    for _ in range(reps):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(graphs) + 1)]
        ev[0].record()
        for i, gr in enumerate(graphs):
            gr.replay()
            ev[i + 1].record()
        torch.cuda.synchronize()
        for i in range(len(graphs)):
            times[i].append(ev[i].elapsed_time(ev[i + 1]))
    if kvr.kvr_sync_status(ctx) != kvr.KVR_OK:
        raise RuntimeError(kvr.kvr_last_error())
    C.close()
    med = [statistics.median(x) / layers for x in times]
    t_app, t_att, t_dec = med[0], med[1], sum(med[2:]) / steps
    kvb = kv_bytes_per_key()
    att_flops = sum(reuse_flops(L, q) for q in qs)
    att_bytes = L * kvb + T * kvb + 2 * T * HQ * D * 2
    dec_flops = sum(4 * HQ * D * (L + q + t + 1) for q in qs for t in range(steps)) / steps
    dec_bytes = L * kvb + sum((q + t + 1) * kvb for q in qs for t in range(steps)) / steps + 2 * B * HQ * D * 2
    tf_att = att_flops / (t_att * 1e-3) / 1e12
    tf_dec = dec_flops / (t_dec * 1e-3) / 1e12
    return {"workload": f"L={L} shared prefix, {B} consumers, suffixes uniform in [16, 512] (total {T} tokens), "
                        f"then {steps} decode steps of all consumers; {layers} layers timed, figures per layer",
            "append_ms_per_layer": t_app, "reuse_ms_per_layer": t_att,
            "reuse_tflops": tf_att, "reuse_frac_bf16_burst": tf_att / peaks["bf16_tflops"],
            "reuse_algorithmic_bytes_per_layer": att_bytes,
            "decode_step_ms_per_layer": t_dec, "decode_tflops": tf_dec,
            "decode_frac_bf16_burst": tf_dec / peaks["bf16_tflops"],
            "decode_gbs_prefix_once": dec_bytes / (t_dec * 1e-3) / 1e9,
            "decode_frac_hbm": dec_bytes / (t_dec * 1e-3) / 1e9 / peaks["hbm_gbs"],
            "decode_tokens_per_s_36_layers": B / (t_dec * 1e-3 * 36),
            "bound": "reuse: tensor (%.0f flop/B); decode: %.0f flop/B" % (att_flops / att_bytes, dec_flops / dec_bytes)}


def run_gpu(args):
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    from paper_2606_13361_gb300 import kvr

    wl = Workload(args, kvr, torch, args.seed + rank)
    n_graphs = len(wl.graphs)
    for _ in range(args.warmup):
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(n_graphs + 1)]
        wl.run_step(evs)
    torch.cuda.synchronize()
    st = kvr.kvr_sync_status(wl.C.ctx)
    if st != kvr.KVR_OK:
        raise RuntimeError(f"device status {st}: {kvr.kvr_last_error()}")

    all_evs = [[torch.cuda.Event(enable_timing=True) for _ in range(n_graphs + 1)]
               for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    sampler = ClockSampler(local)
    sampler.__enter__()
    t_wall = time.perf_counter()
    for evs in all_evs:
        wl.run_step(evs)
    torch.cuda.synchronize()
    t_wall = time.perf_counter() - t_wall
    clocks = sampler.stop()
    if world > 1:
        dist.barrier()
    st = kvr.kvr_sync_status(wl.C.ctx)
    if st != kvr.KVR_OK:
        raise RuntimeError(f"device status {st}: {kvr.kvr_last_error()}")

    K, L, q, nd, NL = args.steps, args.L, args.q, args.decode, args.layers
    total_ms = all_evs[0][0].elapsed_time(all_evs[-1][-1])
    ph = phase_times(wl, all_evs)
    reuse_attn_ms = ph["reuse_attn"] + ph["decode_step"]
    bytes_q = NL * reuse_bytes(L, q)
    bytes_dec = NL * sum(reuse_bytes(L + q + t, 1) for t in range(nd))
    step_reuse_bytes = bytes_q + bytes_dec
    max_ms, units = reduce_over_ranks(reuse_attn_ms, K * step_reuse_bytes)
    max_total, _ = reduce_over_ranks(total_ms, 0.0)
    value = units / (max_ms * 1e-3) / 1e9

    peaks, src = load_peaks()
    pre_ms_per_launch = ph["prefill_attn"] / (K * NL)
    q64_ms = ph["reuse_attn"] / (K * NL)
    dec_ms = ph["decode_step"] / (K * NL * nd)
    pf = prefill_flops(L)
    prefill_tflops = pf / (pre_ms_per_launch * 1e-3) / 1e12
    reuse_gbs_q64 = reuse_bytes(L, q) / (q64_ms * 1e-3) / 1e9
    dec_gbs = (bytes_dec / (NL * nd)) / (dec_ms * 1e-3) / 1e9

    shares = {k: v / total_ms for k, v in ph.items()}
    dominant = max(shares, key=shares.get)
    tr_pre, src_pre = ncu_traffic("prefill")
    tr_dec, src_dec = ncu_traffic("decode")
    tr_q64, src_q64 = ncu_traffic("reuse_q64")
    rf_pre = {"bound": "tensor", "achieved": prefill_tflops, "peak": peaks["bf16_tflops"],
              "unit": "TFLOP/s", "frac": prefill_tflops / peaks["bf16_tflops"],
              "traffic": tr_pre, "traffic_source": src_pre, "kernel": "attn_kernel<128> (kvr_prefill_attn)",
              "per_launch": f"{pf / 1e9:.1f} GFLOP (one layer, L={L})",
              "peak_source": f"{src} bf16_tflops (burst: every timed region here lasts well under a second)"}
    rf_q64 = {"bound": "hbm", "achieved": reuse_gbs_q64, "peak": peaks["hbm_gbs"], "unit": "GB/s",
              "frac": reuse_gbs_q64 / peaks["hbm_gbs"], "traffic": tr_q64, "traffic_source": src_q64,
              "kernel": "attn_kernel<128> + combine_kernel<128> (kvr_reuse_attn, q=64)",
              "per_launch": f"{reuse_bytes(L, q) / 1e6:.2f} MB", "peak_source": f"{src} hbm_gbs"}
    rf_dec = {"bound": "hbm", "achieved": dec_gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
              "frac": dec_gbs / peaks["hbm_gbs"], "traffic": tr_dec, "traffic_source": src_dec,
              "kernel": "decode_kernel<128, fused> (kvr_decode_step)",
              "per_launch": f"{reuse_bytes(L + q, 1) / 1e6:.2f} MB (first step; +4 KB per step)",
              "peak_source": f"{src} hbm_gbs"}
    rf_reuse = {"bound": "hbm", "achieved": value, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": value / peaks["hbm_gbs"], "traffic": None,
                "kernel": "all reuse calls of the step: q=64 attention + 24 decode steps",
                "peak_source": f"{src} hbm_gbs"}
    # Beside each fraction of the measured peak: the fraction of the nominal
    # peak, and t_roof / t (t_roof = max(bytes / HBM, flops / tensor) over the
    # algorithmic work, both at the measured peaks).
    pre_bytes = reuse_bytes(0, L)  # Q, K, V read once, O written: the prefill's own inputs
    q64_flops = reuse_flops(L, q)
    dec_flops = sum(reuse_flops(L + q + t, 1) for t in range(nd)) / nd
    for rf, t_ms, nbytes, flops in ((rf_pre, pre_ms_per_launch, pre_bytes, pf),
                                    (rf_q64, q64_ms, reuse_bytes(L, q), q64_flops),
                                    (rf_dec, dec_ms, bytes_dec / (NL * nd), dec_flops)):
        rf["frac_nominal"] = rf["achieved"] / (NOMINAL_TFLOPS if rf["unit"] == "TFLOP/s" else NOMINAL_GBS)
        t_roof = max(nbytes / (peaks["hbm_gbs"] * 1e9), flops / (peaks["bf16_tflops"] * 1e12))
        rf["t_roof_over_t"] = t_roof / (t_ms * 1e-3)
    rf_reuse["frac_nominal"] = value / NOMINAL_GBS
    by_phase = {"prefill_attn": rf_pre, "reuse_attn": rf_q64, "decode_step": rf_dec}
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": max_total / K, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (torch Philox on device, seeded; N(0,1) q/k/v, norm weights 1+0.1N(0,1))",
        "config": workload_config(args),
        "prefill_attn_tflops": prefill_tflops,
        "reuse_attn_gbs": {"q64": reuse_gbs_q64, "decode": dec_gbs},
        "cost_ratio": {"attn_q64": pre_ms_per_launch / q64_ms, "attn_q1": pre_ms_per_launch / dec_ms,
                       "path_q64": (ph["prefill_append"] + ph["prefill_attn"]) /
                                   (ph["reuse_append"] + ph["reuse_attn"]),
                       "path_q1": (ph["prefill_append"] + ph["prefill_attn"]) / (K * NL) / dec_ms,
                       "note": "attn_*: attention kernels only; path_*: append + attention; the decode "
                               "step (q=1) is one fused append + attention launch"},
        "phase_ms_per_step": {k: v / K for k, v in ph.items()},
        # Sec. 4 on this GPU, whole 36-layer attention path of the document:
        # C_prefill = append + prefill attention over L tokens; C_load = artifact
        # load + one continuation step (q = 64 new tokens, or one decode token)
        "cost_model": {
            "q64": cost_model((ph["prefill_append"] + ph["prefill_attn"]) / K,
                              (ph["load"] + ph["reuse_append"] + ph["reuse_attn"]) / K),
            "q1": cost_model((ph["prefill_append"] + ph["prefill_attn"]) / K,
                             ph["load"] / K + ph["decode_step"] / (K * nd)),
            "paper_m1_L3774": dict(PAPER_M1_L3774, N_star=PAPER_M1_L3774["C_prefill_s"] /
                                   (PAPER_M1_L3774["C_prefill_s"] - PAPER_M1_L3774["C_reuse_s"])),
            "note": "attention path only (no projections or MLP); load = copy of the 556.5 MB artifact from "
                    "device memory"},
        "roofline": by_phase.get(dominant, rf_reuse),
        "roofline_prefill": rf_pre, "roofline_reuse_q64": rf_q64, "roofline_decode": rf_dec,
        "roofline_reuse_all": rf_reuse,
        "dominant_phase": dominant,
        "gpu_launches": wl.launches_per_step * K,
        "clocks": clocks,
        "wall_s": t_wall,
    }
    if not args.no_e2e:
        e2e_ms, h2d, d2h = e2e_run(args, kvr, torch, wl, n_steps=min(5, max(1, K)))
        e2e_ms, _ = reduce_over_ranks(e2e_ms, 0.0)
        line["e2e"] = {"value": world * step_reuse_bytes / (e2e_ms * 1e-3) / 1e9, "unit": "GB/s",
                       "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                       "ms_per_step": e2e_ms,
                       "path": "eager C-ABI calls; the step's inputs go host->device from pinned memory on a "
                               "copy stream (suffix rows, then decode rows during the suffix phase) and the reuse "
                               "outputs come back (suffix outputs during the decode loop), all inside the timed "
                               "region"}
    if not args.no_io:
        io = run_artifact_io(kvr, torch, wl)
        line["artifact_io"] = io
        for enc in ("bf16", "int8"):
            line["cost_model"][f"q64_{enc}_host_load"] = cost_model(
                (ph["prefill_append"] + ph["prefill_attn"]) / K,
                io[f"{enc}_load_pinned_host"]["ms"] + (ph["reuse_append"] + ph["reuse_attn"]) / K)
        line["int8_probe"] = run_int8_probe(kvr, torch)
    if not args.no_sweep:
        line["sweep"] = run_sweep(kvr, torch, peaks, [int(x) for x in args.sweep.split(",")])
    if not args.no_q8:
        line["int8_resident_decode"] = run_q8_resident(kvr, torch, peaks,
                                                       lengths=[int(x) for x in args.q8_lengths.split(",")])
    if not args.no_serving:
        line["serving"] = run_serving(kvr, torch, peaks)
    if not args.no_layer:
        line["whole_layer"] = run_layer_cost(kvr, torch, peaks)
    if not args.no_hotdoc:
        line["hot_document"] = run_hotdoc(kvr, torch, peaks)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        runs, threads = cpu_oracle_sample(L, q, args.seed, budget_s=args.cpu_budget)
        per = statistics.median(runs)
        line["cpu_baseline"] = {
            "value": reuse_bytes(L, q) / per / 1e9, "unit": "GB/s", "cores": threads, "kind": "oracle",
            "sample": f"oracle reuse attention of one layer ({q} rows x {HQ} heads over {L + q} keys, "
                      f"fp64), {len(runs)} runs in {sum(runs):.1f} s, median"}
    if rank == 0:
        print(json.dumps(line))
    wl.C.close()
    if world > 1:
        dist.destroy_process_group()


# --------------------------------------------------------- profiler cases ----

def run_case(args):
    """One call type of the path on a small setup, for a profiler capture (and
    a quick CUDA-event timing): `--case-reps` calls back to back after one
    warm-up call.  Cases: reuse_q64 (q = 64 continuation after L = 3774, one
    layer), decode (fused decode step after L + 64), prefill (L = 3774 prefill
    attention), hotdoc_decode (a B = 256 decode step over a shared L = 32768
    prefix, ragged suffixes uniform in [16, 512], one layer), gemm (the four
    projections of one Qwen3-4B layer over L tokens, each timed).  Prints one
    JSON line with the median per-call time."""
    import torch
    from paper_2606_13361_gb300 import inputs, kvr
    torch.cuda.set_device(0)
    dev = torch.device("cuda")
    g = torch.Generator(device=dev)
    g.manual_seed(args.seed)

    def rn(*shape):
        return torch.randn(shape, generator=g, device=dev).to(torch.bfloat16)
    w = (1.0 + 0.1 * torch.randn((2, D), generator=g, device=dev)).to(torch.bfloat16)
    case, reps = args.case, max(1, args.case_reps)
    if case == "layer_decode":
        # one decode token through `--layers` Qwen3-4B-shaped layers (random
        # weights, more than L2 in all) over an L + q token cache: one CUDA
        # graph of the layer calls, timed, then replayed `reps` times
        NL, T0 = args.layers, args.L + args.q
        H, I = QWEN_HIDDEN, QWEN_INTER
        desc = kvr.make_desc(NL, HQ, HKV, D, max_positions=T0 + 256)
        ld = kvr.kvr_layer_desc(H, I)
        C = kvr.Context(desc, n_pages=2 * (T0 // 128 + 4), max_seqs=4)
        ctx = C.ctx

        def lin(o, i):
            return (torch.randn((o, i), generator=g, device=dev) / math.sqrt(i)).to(torch.bfloat16)

        def nw(n):
            return (1 + 0.1 * torch.randn((n,), generator=g, device=dev)).to(torch.bfloat16)
        Wd = [{"input_norm": nw(H), "wq": lin(HQ * D, H), "wk": lin(HKV * D, H), "wv": lin(HKV * D, H),
               "q_norm": nw(D), "k_norm": nw(D), "wo": lin(H, HQ * D), "post_norm": nw(H),
               "w_gate_up": lin(2 * I, H), "w_down": lin(H, I)} for _ in range(NL)]
        Ws = [kvr.layer_weights(wl) for wl in Wd]
        weight_bytes = sum(t.numel() * 2 for wl in Wd for t in wl.values())
        x = kvr.kvr_seq_open(ctx)
        for l in range(NL):
            qx = torch.empty((T0, HQ, D), dtype=torch.bfloat16, device=dev)
            kvr.kvr_append_kv(ctx, l, [x], [0], [0, T0], rn(T0, HQ, D), rn(T0, HKV, D), rn(T0, HKV, D), w[0], w[1], qx)
            del qx
        kvr.kvr_seq_advance(ctx, [x], [T0])
        kvr.kvr_seq_reserve(ctx, [x], [1])
        ws = torch.empty(kvr.kvr_layer_workspace_bytes(desc, ld, 1), dtype=torch.uint8, device=dev)
        h_t = rn(1, H)
        bufs = [torch.empty((1, H), dtype=torch.bfloat16, device=dev) for _ in range(2)]

        def model():
            src = h_t
            for l in range(NL):
                kvr.kvr_layer_forward(ctx, l, ld, Ws[l], [x], [T0], [0, 1], src, bufs[l % 2], ws)
                src = bufs[l % 2]
        model()
        torch.cuda.synchronize()
        gr = _graph(torch, model)
        t = _time_graph(torch, gr, reps)
        st = kvr.kvr_sync_status(ctx)
        if st != kvr.KVR_OK:
            raise RuntimeError(f"device status {st}: {kvr.kvr_last_error()}")
        C.close()
        kv = NL * reuse_bytes(T0, 1)
        print(json.dumps({"case": case, "layers": NL, "T0": T0, "ms_per_token": t, "us_per_layer": t * 1e3 / NL,
                          "weight_bytes": weight_bytes, "kv_bytes": kv,
                          "gbs": (weight_bytes + kv) / (t * 1e-3) / 1e9,
                          "note": "CUDA graph of the layer calls; not a bench value"}))
        return
    if case == "gemm":
        # the four projections of one Qwen3-4B layer over the L-token document
        T, H, I = args.L, QWEN_HIDDEN, QWEN_INTER
        desc = kvr.make_desc(1, HQ, HKV, D, max_positions=256)
        C = kvr.Context(desc, n_pages=2, max_seqs=2)
        ctx = C.ctx

        def lin(o, i):
            return (torch.randn((o, i), generator=g, device=dev) / math.sqrt(i)).to(torch.bfloat16)
        x, xo, xa = rn(T, H), rn(T, HQ * D), rn(T, I)
        wqkv, wo, wgu, wd = lin(HQ * D + 2 * HKV * D, H), lin(H, HQ * D), lin(2 * I, H), lin(H, I)
        yq = torch.empty((T, HQ * D + 2 * HKV * D), dtype=torch.bfloat16, device=dev)
        yo, yd = torch.empty((T, H), dtype=torch.bfloat16, device=dev), torch.empty((T, H), dtype=torch.bfloat16, device=dev)
        ya = torch.empty((T, I), dtype=torch.bfloat16, device=dev)
        calls = {"qkv": (lambda: kvr.kvr_linear(ctx, x, wqkv, yq), 2 * T * H * (HQ * D + 2 * HKV * D)),
                 "o": (lambda: kvr.kvr_linear(ctx, xo, wo, yo, x), 2 * T * HQ * D * H),
                 "gate_up_swiglu": (lambda: kvr.kvr_linear_swiglu(ctx, x, wgu, ya), 2 * T * H * 2 * I),
                 "down": (lambda: kvr.kvr_linear(ctx, xa, wd, yd, x), 2 * T * I * H)}
        res = {}
        for name, (fn, flops) in calls.items():
            fn()
            torch.cuda.synchronize()
            ts = []
            for _ in range(reps):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                fn()
                e1.record()
                torch.cuda.synchronize()
                ts.append(e0.elapsed_time(e1) * 1e3)
            t = statistics.median(ts)
            res[name] = {"us": t, "tflops": flops / (t * 1e-6) / 1e12}
        st = kvr.kvr_sync_status(ctx)
        if st != kvr.KVR_OK:
            raise RuntimeError(f"device status {st}: {kvr.kvr_last_error()}")
        C.close()
        print(json.dumps({"case": case, "T": T, "reps": reps, "gemms": res,
                          "note": "eager calls, one launch each; not a bench value"}))
        return
    if case == "hotdoc_decode":
        L, B, steps = 32768, 256, reps + 1
        qs = [int(x) for x in inputs.ragged_lengths(3, B, 16, 512)]
        T = sum(qs)
        desc = kvr.make_desc(1, HQ, HKV, D, max_positions=L + 512 + steps + 256)
        C = kvr.Context(desc, n_pages=(L + 127) // 128 + B * ((512 + steps + 127) // 128 + 1) + 8, max_seqs=B + 4)
        ctx = C.ctx
        art = rn(kvr.kvr_artifact_bytes(desc, L) // 2)
        p = kvr.kvr_load_kv(ctx, kvr.kvr_artifact_meta(desc.model_id, 1, L), art, True)
        seqs = [kvr.kvr_seq_fork(ctx, p) for _ in range(B)]
        cu = [0]
        for q in qs:
            cu.append(cu[-1] + q)
        qo = torch.empty((T, HQ, D), dtype=torch.bfloat16, device=dev)
        kvr.kvr_append_kv(ctx, 0, seqs, [L] * B, cu, rn(T, HQ, D), rn(T, HKV, D), rn(T, HKV, D), w[0], w[1], qo)
        kvr.kvr_seq_advance(ctx, seqs, qs)
        kvr.kvr_seq_reserve(ctx, seqs, [steps] * B)
        dec = (rn(B, HQ, D), rn(B, HKV, D), rn(B, HKV, D))
        dq, do = torch.empty((B, HQ, D), dtype=torch.bfloat16, device=dev), torch.empty((B, HQ, D), dtype=torch.bfloat16, device=dev)
        pos = [L + q for q in qs]

        def call():
            kvr.kvr_decode_step(ctx, 0, seqs, pos, list(range(B + 1)), *dec, w[0], w[1], dq, do)
            kvr.kvr_seq_advance(ctx, seqs, [1] * B)
            for i in range(B):
                pos[i] += 1
    else:
        L, q = args.L, args.q
        desc = kvr.make_desc(1, HQ, HKV, D, max_positions=L + q + reps + 256)
        C = kvr.Context(desc, n_pages=3 * ((L + q + reps) // 128 + 4), max_seqs=8)
        ctx = C.ctx
        x = kvr.kvr_seq_open(ctx)
        qx = torch.empty((L, HQ, D), dtype=torch.bfloat16, device=dev)
        kvr.kvr_append_kv(ctx, 0, [x], [0], [0, L], rn(L, HQ, D), rn(L, HKV, D), rn(L, HKV, D), w[0], w[1], qx)
        ox = torch.empty_like(qx)
        if case == "prefill":
            def call():
                kvr.kvr_prefill_attn(ctx, 0, x, L, qx, ox)
        else:
            kvr.kvr_seq_advance(ctx, [x], [L])
            c = kvr.kvr_seq_fork(ctx, x)
            qs_ = torch.empty((q, HQ, D), dtype=torch.bfloat16, device=dev)
            kvr.kvr_append_kv(ctx, 0, [c], [L], [0, q], rn(q, HQ, D), rn(q, HKV, D), rn(q, HKV, D), w[0], w[1], qs_)
            os_ = torch.empty_like(qs_)
            if case == "reuse_q64":
                def call():
                    kvr.kvr_reuse_attn(ctx, 0, [c], [0, q], qs_, os_)
            elif case == "decode":
                kvr.kvr_seq_advance(ctx, [c], [q])
                kvr.kvr_seq_reserve(ctx, [c], [reps + 1])
                dec = (rn(1, HQ, D), rn(1, HKV, D), rn(1, HKV, D))
                od = torch.empty((1, HQ, D), dtype=torch.bfloat16, device=dev)
                pos = [L + q]

                def call():
                    kvr.kvr_decode_step(ctx, 0, [c], pos, [0, 1], *dec, w[0], w[1], None, od)
                    kvr.kvr_seq_advance(ctx, [c], [1])
                    pos[0] += 1
            else:
                raise SystemExit(f"unknown case {case}")
    call()
    torch.cuda.synchronize()
    times = []
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        call()
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1) * 1e3)
    st = kvr.kvr_sync_status(ctx)
    if st != kvr.KVR_OK:
        raise RuntimeError(f"device status {st}: {kvr.kvr_last_error()}")
    C.close()
    print(json.dumps({"case": case, "reps": reps, "us_per_call_median": statistics.median(times),
                      "note": "eager calls (launch overhead included); not a bench value"}))


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["kvr", "reference"], default="kvr")
    ap.add_argument("--layers", type=int, default=36)
    ap.add_argument("--L", type=int, default=3774)
    ap.add_argument("--q", type=int, default=64)
    ap.add_argument("--decode", type=int, default=24)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-budget", type=float, default=10.0)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sweep", action="store_true", help="skip the L sweep (prefill vs reuse per L)")
    ap.add_argument("--sweep", default="1024,2048,4096,8192,16384,32768")
    ap.add_argument("--no-serving", action="store_true", help="skip the 64-consumer shared-prefix section")
    ap.add_argument("--no-q8", action="store_true", help="skip decode over int8-resident prefixes")
    ap.add_argument("--q8-lengths", default="3838,32768", help="contexts of the int8-resident decode section")
    ap.add_argument("--no-io", action="store_true", help="skip the artifact load/export transfer rates")
    ap.add_argument("--no-layer", action="store_true", help="skip the 36-layer whole-model cost section")
    ap.add_argument("--no-hotdoc", action="store_true", help="skip the 256-consumer 32K hot-document section")
    ap.add_argument("--case", default=None, help="run one call type for a profiler capture instead of the bench "
                                                 "(reuse_q64, decode, prefill, hotdoc_decode, gemm)")
    ap.add_argument("--case-reps", type=int, default=3)
    args = ap.parse_args(argv)
    if args.case:
        run_case(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
