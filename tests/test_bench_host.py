"""Host-side logic of bench.py: the algorithmic byte/flop counts the roofline
uses, and the max-time / summed-units reduction over ranks (gloo, 2 ranks)."""
import os
import socket

import pytest
import torch.multiprocessing as mp

import bench


def test_algorithmic_counts_match_the_workload_arithmetic():
    # Qwen3-4B layer: 8 KV heads x 128 x 2 (K, V) x 2 B = 4096 B per key
    assert bench.kv_bytes_per_key() == 4096
    # reuse q=64 after L=3774: 3838 keys once + Q and O (64 x 32 x 128 x 2 B each)
    assert bench.reuse_bytes(3774, 64) == 3838 * 4096 + 2 * 64 * 32 * 128 * 2
    assert abs(bench.reuse_bytes(3774, 64) / 1e6 - 16.77) < 0.01
    # causal prefill: 4 Hq d per (row, visible key) pair, L(L+1)/2 pairs
    assert abs(bench.prefill_flops(3774) / 1e9 - 116.7) < 0.1
    assert bench.prefill_flops(1) == 4 * 32 * 128
    assert bench.reuse_flops(0, 3) == bench.prefill_flops(3)


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    t, u = bench.reduce_over_ranks(10.0 + rank, 100.0 * (rank + 1))
    out.put((rank, t, u))
    dist.destroy_process_group()


def test_reduce_over_ranks_gloo_two_ranks():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # elapsed = max over ranks, units summed (weak scaling: every rank runs a replica)
    assert res == [(0, 11.0, 300.0), (1, 11.0, 300.0)]


def test_single_process_reduction_is_identity():
    assert bench.reduce_over_ranks(3.5, 7.0) == (3.5, 7.0)


def test_reference_arm_prints_a_bounded_line(capsys):
    bench.main(["--impl", "reference", "--steps", "1", "--warmup", "0", "--L", "300", "--q", "8"])
    import json
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["unit"] == "GB/s" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0


def test_cost_model_follows_eqs_1_to_3():
    """bench's cost model (Sec. 4) agrees with the oracle's Eqs. 1-3 and with
    the paper's Table 1 reading: 14.71 s prefill vs 0.296 s reuse at L = 3774
    gives a break-even just above one reuse."""
    import oracle
    cm = bench.cost_model(120.0, 3.0, ns=(1, 7, 1000))
    assert cm["N_star"] == oracle.break_even(120.0, 3.0)
    flat, reuse = oracle.per_call_cost(120.0, 3.0, [1, 7, 1000])
    for i, n in enumerate((1, 7, 1000)):
        assert cm["per_call_ms"][str(n)]["from_scratch"] == flat[i]
        assert abs(cm["per_call_ms"][str(n)]["kv_reuse"] - reuse[i]) < 1e-12
    assert cm["saving_ms_at_1000"] == 1000 * (120.0 - 3.0)
    assert bench.cost_model(5.0, 0.0)["N_star"] == 1.0
    m1 = bench.PAPER_M1_L3774
    assert 1.02 <= m1["C_prefill_s"] / (m1["C_prefill_s"] - m1["C_reuse_s"]) <= 1.13


def test_ncu_traffic_is_reported_only_for_the_captured_sources(tmp_path, monkeypatch):
    """bench.ncu_traffic returns a capture's per-launch DRAM bytes only while
    the kernel sources hash to the value recorded with the capture."""
    for kind, rec in bench.NCU_TRAFFIC.items():
        assert rec["source"].startswith("profiles/") and os.path.exists(os.path.join(bench.ROOT, rec["source"]))
        got, src = bench.ncu_traffic(kind)
        assert src == rec["source"]
        assert got in (None, rec["bytes"])
    # a changed source file makes the recorded figure stale
    csrc = tmp_path / "paper_2606_13361_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for f in bench.NCU_TRAFFIC["decode"]["files"]:
        (csrc / f).write_bytes(b"changed")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.ncu_traffic("decode")[0] is None


def test_stage_summary_of_a_synthetic_trace():
    """stage_trace.summarise: per-stage median / p10 / p90 over CTAs and
    layers, relative to each CTA's grid-dependency stamp, plus the spread of
    those stamps within a launch and the launch period."""
    import numpy as np
    from paper_2606_13361_gb300 import stage_trace
    layers, ctas = 4, 10
    buf = np.zeros((40, 160, 32), dtype=np.uint64)
    for l in range(layers):
        for c in range(ctas):
            t1 = 1_000_000 + 7_500 * l + 30 * c  # ns: launch period 7.5 us, 30 ns apart
            buf[l, c, 0] = t1 - 500
            buf[l, c, 1] = t1
            buf[l, c, 2] = t1 + 1_500 + 10 * c
            buf[l, c, 21] = t1 + 6_000
    out = stage_trace.summarise(buf, layers, {2: "prologue done", 21: "end"})
    assert out["ctas"] == ctas
    assert out["end"] == [6.0, 6.0, 6.0]
    med, p10, p90 = out["prologue done"]
    assert 1.5 <= p10 <= med <= p90 <= 1.6
    assert out["launch period"] == 7.5
    assert out["grid dependency spread over a launch"] == 0.27
