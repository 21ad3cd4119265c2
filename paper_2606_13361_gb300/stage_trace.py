"""Stage timing of the hot kernels and instruction-rate probes (latency analysis).

Builds a variant of the library with KVR_STAGE_TRACE defined (every CTA of the
decode and attention kernels stores %globaltimer at the stages listed in their
sources) plus the rate probes of csrc/kvr_probe.cu, into _build_trace/ and
libkvr_trace.so beside the package; libkvr.so is not touched.  Then, on
cuda:0:

  python -m paper_2606_13361_gb300.stage_trace decode  --L 3838   # 36-layer graph of decode steps
  python -m paper_2606_13361_gb300.stage_trace reuse   --L 3774 --B 1 --q 64
  python -m paper_2606_13361_gb300.stage_trace prefill --L 3774
  python -m paper_2606_13361_gb300.stage_trace rates              # mma.sync and ex2 rates
  python -m paper_2606_13361_gb300.stage_trace copies             # 16 KB copy latency by route

Each workload prints one JSON line: the per-call time of the graph and, per
stage, the median (p10, p90) over CTAs and layers of the time after the CTA's
grid dependency resolved, in microseconds.  The stamps cost a global store
each, so the traced calls run a little slower than the product's.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import sys

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
TRACE_LIB = os.path.join(_PKG, "libkvr_trace.so")
HQ, HKV, D = 32, 8, 128  # Qwen3-4B attention shapes

DECODE_STAGES = {2: "prologue done", 3: "warp 0's first unit landed", 16: "warp 0's units done",
                 17: "warp states stored", 18: "cluster merge start", 19: "partials pushed",
                 20: "partials received", 21: "end"}
# 6-warp CTAs only: the prologue's parts and each warp's two units
DECODE_STAGES_6 = {28: "first copies issued (warp 0)", 29: "q/k norm + RoPE done (last warp)",
                   30: "q fragments loaded (warp 0)", 31: "warp 0's first copy landed (polled)"}
DECODE_STAGES_6.update({4 + w: f"warp {w}: last unit done" for w in range(6)})
DECODE_STAGES_6.update({10 + w: f"warp {w}: first unit done" for w in range(6)})
DECODE_STAGES_6.update({22 + w: f"warp {w}: second unit landed" for w in range(6)})
ATTN_STAGES = {2: "Q and first K tile landed", 3: "first P stored", 4: "last P stored",
               5: "waiting for the last P V", 6: "output stored", 7: "end"}
ATTN_STAGES.update({8 + j: f"warpgroup 0: P of key tile {j} stored" for j in range(10)})
ATTN_STAGES.update({18 + j: f"warpgroup 1: P of key tile {j} stored" for j in range(10)})
ATTN_STAGES.update({28: "last P V done (warpgroup 0)", 29: "row sums exchanged", 30: "partial staged in shared memory"})
# two Q tiles per CTA (prefill): the hops around key tile 4 / 5 of Q tile A
PREFILL_STAGES = {k: v for k, v in ATTN_STAGES.items() if k < 18}
PREFILL_STAGES.update({k: f"warpgroup 0, warp {k - 24}: P of key tile 4 stored" for k in range(24, 28)})
PREFILL_STAGES.update({28: "MMA warp: V(4) landed", 29: "MMA warp: P_A(4) seen",
                       30: "MMA warp: P_A V_4 issued", 31: "softmax A: S_A(5) seen"})


def build(verbose=False) -> str:
    from . import build as b
    return b.build_library(verbose=verbose, defines=("KVR_STAGE_TRACE",), extra_sources=("kvr_probe.cu",),
                           build_dir=os.path.join(_PKG, "_build_trace"), lib=TRACE_LIB)


def _kvr():
    from . import kvr
    kvr.LIB_PATH = TRACE_LIB
    kvr.lib = kvr._load()
    return kvr


def _graph_us(torch, fn, layers, reps=8):
    fn()
    torch.cuda.synchronize()
    gr = torch.cuda.CUDAGraph()
    st = torch.cuda.Stream()
    st.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(st):
        with torch.cuda.graph(gr, stream=st):
            fn()
    torch.cuda.current_stream().wait_stream(st)
    torch.cuda.synchronize()
    ts = []
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        gr.replay()
        e1.record()
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1) * 1e3 / layers)
    return float(np.median(ts))


def summarise(buf, layers, stages):
    """Stage times after each CTA's grid dependency (slot 1), in us."""
    t = buf[:layers].astype(np.int64)
    live = t[0, :, 0] > 0
    t = t[:, live]
    out = {"ctas": int(live.sum())}
    rel = t[:, :, 1]
    for slot, name in stages.items():
        v = (t[:, :, slot] - rel) / 1e3
        v = v[(t[:, :, slot] > 0) & (np.abs(v) < 1e4)]
        if v.size:
            out[name] = [round(float(np.median(v)), 2), round(float(np.percentile(v, 10)), 2),
                         round(float(np.percentile(v, 90)), 2)]
    first = rel.min(axis=1)
    out["grid dependency spread over a launch"] = round(float(np.median(rel.max(axis=1) - first)) / 1e3, 2)
    out["launch period"] = round(float(np.median(np.diff(first))) / 1e3, 2)
    return out


def _context(kvr, torch, L, layers, extra_pages, max_seqs):
    desc = kvr.make_desc(layers, HQ, HKV, D, max_positions=L + 1024)
    C = kvr.Context(desc, n_pages=2 * ((L + 127) // 128) + 8 + extra_pages, max_seqs=max_seqs)
    g = torch.Generator(device="cuda")
    g.manual_seed(1)

    def rn(*s):
        return torch.randn(s, generator=g, device="cuda").to(torch.bfloat16)
    w = (1.0 + 0.1 * torch.randn((2, D), generator=g, device="cuda")).to(torch.bfloat16)
    x = kvr.kvr_seq_open(C.ctx)
    pre = (rn(L, HQ, D), rn(L, HKV, D), rn(L, HKV, D))
    qx = torch.empty((L, HQ, D), dtype=torch.bfloat16, device="cuda")
    return C, rn, w, x, pre, qx


def run_decode(args):
    import torch
    kvr = _kvr()
    L, NL = args.L, args.layers
    C, rn, w, x, pre, qx = _context(kvr, torch, L, NL, 0, 8)
    ctx = C.ctx
    for l in range(NL):
        kvr.kvr_append_kv(ctx, l, [x], [0], [0, L], *pre, w[0], w[1], qx)
    kvr.kvr_seq_advance(ctx, [x], [L])
    c = kvr.kvr_seq_fork(ctx, x)
    dq, dk, dv = rn(1, HQ, D), rn(1, HKV, D), rn(1, HKV, D)
    od = torch.empty((NL, 1, HQ, D), dtype=torch.bfloat16, device="cuda")
    us = _graph_us(torch, lambda: [kvr.kvr_decode_step(ctx, l, [c], [L], [0, 1], dq, dk, dv, w[0], w[1], None, od[l])
                                   for l in range(NL)], NL)
    buf = np.zeros((40, 160, 32), dtype=np.uint64)
    assert kvr.lib.kvr_stage_read_decode(ctypes.c_void_p(buf.ctypes.data), buf.nbytes) == 0
    assert kvr.kvr_sync_status(ctx) == kvr.KVR_OK
    st = summarise(buf, NL, DECODE_STAGES)
    if args.detail:
        st["detail (6-warp CTAs)"] = summarise(buf, NL, DECODE_STAGES_6)
    return {"workload": f"decode step after L={L}, {NL}-layer graph", "us_per_call": round(us, 3), "stages_us": st}


def run_attention(args, prefill):
    import torch
    kvr = _kvr()
    L, NL, B, q = args.L, args.layers, args.B, args.q
    C, rn, w, x, pre, qx = _context(kvr, torch, L, NL, 2 * B, max(8, B + 2))
    ctx = C.ctx
    for l in range(NL):
        kvr.kvr_append_kv(ctx, l, [x], [0], [0, L], *pre, w[0], w[1], qx)
    if prefill:
        ox = torch.empty_like(qx)
        us = _graph_us(torch, lambda: [kvr.kvr_prefill_attn(ctx, l, x, L, qx, ox) for l in range(NL)], NL)
        name = f"prefill attention, L={L}, {NL}-layer graph"
    else:
        kvr.kvr_seq_advance(ctx, [x], [L])
        cs = [kvr.kvr_seq_fork(ctx, x) for _ in range(B)]
        suf = (rn(B * q, HQ, D), rn(B * q, HKV, D), rn(B * q, HKV, D))
        qs = [torch.empty((B * q, HQ, D), dtype=torch.bfloat16, device="cuda") for _ in range(NL)]
        os_ = [torch.empty((B * q, HQ, D), dtype=torch.bfloat16, device="cuda") for _ in range(NL)]
        cu = [i * q for i in range(B + 1)]
        for l in range(NL):
            kvr.kvr_append_kv(ctx, l, cs, [L] * B, cu, *suf, w[0], w[1], qs[l])
        us = _graph_us(torch, lambda: [kvr.kvr_reuse_attn(ctx, l, cs, cu, qs[l], os_[l]) for l in range(NL)], NL)
        name = f"reuse attention, {B} consumer(s) x q={q} after L={L}, {NL}-layer graph"
    buf = np.zeros((40, 160, 32), dtype=np.uint64)
    assert kvr.lib.kvr_stage_read_attn(ctypes.c_void_p(buf.ctypes.data), buf.nbytes) == 0
    assert kvr.kvr_sync_status(ctx) == kvr.KVR_OK
    st = summarise(buf, NL, PREFILL_STAGES if prefill else ATTN_STAGES)
    # steady-state interval between a warpgroup's P stores of consecutive key
    # tiles (tiles 2..9 of CTAs that reach them)
    t = buf[:NL].astype(np.int64)
    for wg in ((0,) if prefill else (0, 1)):  # (two Q tiles: warpgroup 0 only)
        p_ = t[:, :, 8 + 10 * wg + 2:8 + 10 * wg + 10]
        dv = np.diff(p_, axis=2) / 1e3
        ok = (p_[:, :, 1:] > 0) & (p_[:, :, :-1] > 0)
        if ok.any():
            st[f"warpgroup {wg}: us between P stores of consecutive key tiles"] = round(float(np.median(dv[ok])), 3)
    if prefill:
        st["hops around key tile 4 / 5 of Q tile A"] = prefill_hops(t)
    return {"workload": name, "us_per_call": round(us, 3), "stages_us": st}


def prefill_hops(t):
    """Intervals between the prefill stamps of one CTA around key tile 4 / 5 of
    Q tile A (slots 12, 13: warp 0's P stores of tiles 4 and 5; 24-27: each
    warp of warpgroup 0 stored P of tile 4; 28: the MMA warp has V(4); 29: it
    saw P-full; 30: it issued P_A V_4; 31: softmax A saw S_A(5)), median (p10,
    p90) in us over the CTAs that reach tile 5."""
    need = [12, 13, 24, 25, 26, 27, 28, 29, 30, 31]
    ok = np.all(t[:, :, need] > 0, axis=2)
    if not ok.any():
        return {}
    w = t[:, :, 24:28]
    first, last = w.min(axis=2), w.max(axis=2)

    def d(x, y):
        v = (y - x)[ok] / 1e3
        return [round(float(np.median(v)), 3), round(float(np.percentile(v, 10)), 3),
                round(float(np.percentile(v, 90)), 3)]
    return {"first to last warp of the warpgroup storing P(4)": d(first, last),
            "last warp's P(4) -> MMA warp sees P-full": d(last, t[:, :, 29]),
            "MMA warp has V(4) -> sees P-full": d(t[:, :, 28], t[:, :, 29]),
            "sees P-full -> P_A V_4 issued (8 MMAs)": d(t[:, :, 29], t[:, :, 30]),
            "last warp's P(4) -> softmax sees S_A(5)": d(last, t[:, :, 31]),
            "softmax sees S_A(5) -> warp 0 stores P(5)": d(t[:, :, 31], t[:, :, 13]),
            "warp 0: P(4) -> P(5)": d(t[:, :, 12], t[:, :, 13])}


def run_rates():
    kvr = _kvr()
    f = kvr.lib.kvr_probe_rate
    f.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.POINTER(ctypes.c_ulonglong)]
    f.restype = ctypes.c_int
    iters = 4096
    res = {}

    def probe(kind, warps, chains):
        cyc = ctypes.c_ulonglong(0)
        assert f(kind, warps, chains, iters, ctypes.byref(cyc)) == 0
        return cyc.value
    c = probe(0, 1, 1)
    res["mma.sync m16n8k16 bf16: latency (cycles)"] = round(c / iters, 1)
    c = probe(0, 12, 4)
    res["mma.sync m16n8k16 bf16: per SM, 12 warps x 4 chains (cycles per MMA)"] = round(c / (iters * 48), 2)
    res["mma.sync m16n8k16 bf16: flop/clk/SM"] = round(iters * 48 * 4096 / c)
    c = probe(1, 16, 8)
    res["ex2.approx.f32: results/clk/SM (16 warps)"] = round(iters * 8 * 32 * 16 / c, 2)
    c = probe(2, 16, 8)
    res["ex2.approx.f16x2: results/clk/SM (16 warps)"] = round(2 * iters * 8 * 32 * 16 / c, 2)
    return {"workload": "instruction rates on one SM (clock64)", "rates": res}


def run_copies(args):
    kvr = _kvr()
    f = kvr.lib.kvr_probe_copy
    f.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.POINTER(ctypes.c_ulonglong)]
    f.restype = ctypes.c_int
    n = args.ctas
    res = {}
    for kind, name in enumerate(["TMA tiles (4 x 4 KB)", "cp.async 16 B", "ld.global 16 B into registers",
                                 "bulk copy (2 x 8 KB)", "TMA tiles 5 us after a bulk L2 prefetch",
                                 "TMA tiles 5 us after tensor-tile L2 prefetches",
                                 "TMA tiles 5 us after per-line L2 prefetches"]):
        for warm in ((1, 0) if kind < 4 else (0,)):
            out = (ctypes.c_ulonglong * n)()
            assert f(kind, warm, n, out) == 0
            v = np.array(out[:], dtype=np.float64) / 1e3
            res[f"{name}, {'L2' if warm else 'DRAM'}"] = [round(float(np.median(v)), 3),
                                                          round(float(np.percentile(v, 10)), 3),
                                                          round(float(np.percentile(v, 90)), 3)]
    return {"workload": f"one 16 KB block per one-warp CTA, {n} CTAs: us from issue to arrival, median (p10, p90)",
            "copies_us": res}


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("what", choices=["decode", "reuse", "prefill", "rates", "copies"])
    ap.add_argument("--ctas", type=int, default=96, help="copies: CTAs per launch")
    ap.add_argument("--L", type=int, default=3774)
    ap.add_argument("--B", type=int, default=1)
    ap.add_argument("--q", type=int, default=64)
    ap.add_argument("--layers", type=int, default=36)
    ap.add_argument("--detail", action="store_true", help="decode: per-warp unit and prologue stages")
    args = ap.parse_args(argv)
    build()
    import torch
    torch.cuda.set_device(0)
    if args.what == "decode":
        out = run_decode(args)
    elif args.what == "rates":
        out = run_rates()
    elif args.what == "copies":
        out = run_copies(args)
    else:
        out = run_attention(args, args.what == "prefill")
    print(json.dumps(out))


if __name__ == "__main__":
    sys.exit(main())
