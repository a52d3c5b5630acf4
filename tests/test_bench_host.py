"""Host-side logic of bench.py: the max-over-ranks / sum-over-ranks timing
reduction on world_size 2 over gloo, argument defaults, the attention
roofline arithmetic, the source-keyed DRAM traffic and the clock summary."""
from __future__ import annotations

import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        elapsed = [3.0, 5.0][rank]
        mx = bench.max_over_ranks(elapsed, world)
        tot = bench.sum_over_ranks(100.0 * (rank + 1), world)
        bench.barrier(world)
        q.put((rank, mx, tot))
    finally:
        dist.destroy_process_group()


def test_rank_reductions_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [5.0, 5.0]      # the slowest rank sets the time
    assert [r[2] for r in res] == [300.0, 300.0]  # bytes of all ranks add up


def test_single_process_reductions_are_identity():
    assert bench.max_over_ranks(2.5, 1) == 2.5
    assert bench.sum_over_ranks(2.5, 1) == 2.5


def test_defaults():
    a = bench.parse_args([])
    assert a.gpus == 1 and a.impl == "ours" and a.warmup >= 3 and a.workload == bench.DEFAULT_WORKLOAD


def test_attention_roofline_arithmetic():
    """The roofline object: achieved GB/s = cache bytes read once per launch
    over the launch time; FLOPs count every (query row, visible key) pair,
    the visible keys enumerated here from the causal mask position by
    position; the ridge-aware fraction is the larger of the byte and FLOP
    floors over the measured time."""
    from paper_2607_27269_gb300 import workloads as wl
    s = wl.SHAPES["llama1b_paged_b128_h32_r512_t128_8192"]
    w = wl.make(s, seed=0, batch=3, kv_range=(10, 40))
    peaks = {"hbm_gbs": 5000.0, "bf16_tflops": 2000.0, "source": "test"}
    ms = 0.01
    r = bench.attention_roofline(w, ms, peaks)
    nbytes = sum(int(k) for k in w.kv_len) * (s.rank + s.d_rope) * 2
    assert r["bytes_per_launch"] == nbytes
    assert r["achieved"] == round(nbytes / (ms * 1e-3) / 1e9, 1)
    assert r["frac"] == round(nbytes / (ms * 1e-3) / 1e9 / 5000.0, 4)
    # query i of a sequence whose new entries start at start_pos sees positions p <= start_pos + i
    pairs = 0
    for k, sp in zip(w.kv_len.tolist(), w.start_pos.tolist()):
        for i in range(s.q_len):
            pairs += sum(1 for p in range(k) if p <= sp + i)
    pairs *= s.num_heads
    flops = pairs * (2 * (s.rank + s.d_rope) + 2 * s.rank)
    assert r["flops_per_launch"] == flops
    floor_s = max(nbytes / 5000e9, flops / 2000e12)
    assert r["ridge_frac"] == round(floor_s / (ms * 1e-3), 4)
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["peak"] == 5000.0


def test_attention_traffic_follows_the_kernel_source(monkeypatch):
    """DRAM traffic is reported only for the kernel source it was captured
    from: any other source hash gives null."""
    import hashlib
    with open(os.path.join(bench.ROOT, "paper_2607_27269_gb300", "csrc", "attn_tc.cu"), "rb") as f:
        current = hashlib.sha256(f.read()).hexdigest()[:16]
    name = "llama1b_paged_b128_h32_r512_t128_8192"
    monkeypatch.setattr(bench, "TRAFFIC_SOURCE", current)
    assert bench.attn_traffic(name) == bench.TRAFFIC[name]
    assert bench.attn_traffic("tiny_b1_h8_r128_t256") is None  # never captured
    monkeypatch.setattr(bench, "TRAFFIC_SOURCE", "0" * 16)
    assert bench.attn_traffic(name) is None


def test_clock_summary_flags_throttle_reasons():
    """The clocks object: median SM clock under load, the maximum clock, and
    every throttle reason seen active in any sample (the active-mask column
    itself is not a reason)."""
    import tempfile
    fd, path = tempfile.mkstemp(suffix=".csv")
    with os.fdopen(fd, "w") as f:
        f.write("0, 2070, 2070, 900.5, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active\n")
        f.write("0, 1980, 2070, 1390.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active\n")
        f.write("0, 2055, 2070, 1100.0, 0x0000000000000008, Active, Not Active, Not Active, Not Active\n")
        f.write("garbage line\n")
    c = bench.ClockSampler(0)
    c.proc = object()  # as if nvidia-smi had been started
    c.path = path
    out = c.summary()
    assert out["sm_mhz"] == 2055.0 and out["sm_max_mhz"] == 2070.0 and out["samples"] == 3
    assert out["reasons"] == ["hw_slowdown", "sw_power_cap"]
    assert not os.path.exists(path)
