#!/usr/bin/env python3
"""Benchmark of the absorbed-MLA decode step on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Prints ONE JSON line (rank 0).  A step is one pass of the whole decode path
over one batch: cache append of this step's q_len entries, query absorption,
split-KV attention over the latent cache, split combine, W_UV (and W_O)
projection.  `value` is latent-cache throughput in GB/s (cache bytes the step
must read / step time) with every input resident in HBM; the step replays as a
CUDA graph and rotates over enough replicas of the inputs that the bytes
touched between two reuses exceed twice the L2.  `roofline` rates the
attention kernel (the dominant one) on its own launches, timed with CUDA
events on its stream.  `e2e` repeats the step through the public API with the
step's inputs copied from pinned host memory and the output read back, in the
faster (tried briefly before the timed region) of two loops: a second stream
uploading the next step's inputs and reading this step's output back while it
computes (a serving loop's overlap), or the copies in line on the step's
stream (fewer host calls, for steps too short to hide them).  The step itself
is the public DecodeStep in its CUDA-graph mode (one graph launch per step)
unless --no-graph.
`cpu_baseline` (rank 0, N = 1) times the fp64 CPU oracle on a bounded sample.

Under torchrun (N > 1) every rank runs its own replica of the workload on its
own GPU (weak scaling, no collective on the data path); the timing is the
maximum over ranks and `value` sums the bytes of all ranks.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "llama1b_paged_b128_h32_r512_t128_8192"
# the other workload the attention target names; its attention core is rated in the same run
LONG_WORKLOAD = "llama3b_long_b8_h24_r512_t16k_32k"
METRIC = "MLA decode-attn μs/step and latent-cache HBM GB/s (% of GB300 peak), 1 GPU"
NOMINAL_HBM_GBS = 8000.0  # the ~8 TB/s HBM3e figure the attention target is also quoted against


def parse_args(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--workload", default=DEFAULT_WORKLOAD)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--num-splits", type=int, default=0)
    p.add_argument("--no-graph", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-long", action="store_true",
                   help="skip the second attention rating on the long-context workload")
    p.add_argument("--seed", type=int, default=0)
    p.add_argument("--attn-launches", type=int, default=0,
                   help="profiling aid: one full step, then this many attention launches alone; no timing")
    p.add_argument("--proj-launches", type=int, default=0,
                   help="profiling aid: this many launches of the projection (mla_project_append) alone; no timing")
    p.add_argument("--accept-launches", type=int, default=0,
                   help="profiling aid: this many launches of the acceptance statistics alone; no timing")
    p.add_argument("--gqa-launches", type=int, default=0,
                   help="profiling aid: this many launches of the original-GQA attention alone; no timing")
    return p.parse_args(argv)


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(value: float, world: int, device=None) -> float:
    """Largest value over all ranks (the slowest rank sets the job's time)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value: float, world: int, device=None) -> float:
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ---------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms in the background."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None
        self.t0 = self.t1 = None

    def start(self):
        fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (FileNotFoundError, OSError):
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[4:9]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["active_mask", "hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i in range(1, 5) if r[i].lower().startswith("active")})
        sm = sorted(x[0] for x in rows)
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(x[1] for x in rows), "reasons": reasons,
                "samples": len(rows)}


# ---------------------------------------------------------------- our arm

def run_ours(args, rank, world, local):
    import torch
    from paper_2607_27269_gb300 import abi
    from paper_2607_27269_gb300 import workloads as wl

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    abi.lib()
    shape = wl.SHAPES[args.workload]
    w = wl.make(shape, seed=args.seed + rank)
    cache_bytes = w.cache_bytes
    props = torch.cuda.get_device_properties(dev)
    l2 = getattr(props, "L2_cache_size", 126 * 2 ** 20)
    # bytes one step touches: the cache it reads plus the query / weight / output tensors
    per_replica = (w.c_kv.numel() + w.k_rope.numel()) * 2 + sum(
        t.numel() * t.element_size() for t in (w.w_uk, w.w_uv, w.q_nope, w.q_pe, w.c_new, w.kr_new)
        if t is not None) + (w.w_o.numel() * 2 if w.w_o is not None else 0)
    replicas = max(2, math.ceil(2 * l2 / per_replica) + 1)
    dws = [abi.to_device(w, dev) for _ in range(replicas)]
    steps = [abi.DecodeStep(d.dims, d.cache, d.batch, d.q_len, d.max_kv_len, args.num_splits) for d in dws]
    S = steps[0].num_splits

    def run(i):
        d, st = dws[i % replicas], steps[i % replicas]
        return st(d.q_nope, d.q_pe, d.kv_len, d.w_uk, d.w_uv, d.w_o, c_new=d.c_new, kr_new=d.kr_new,
                  start_pos=d.start_pos)

    stream = torch.cuda.Stream(dev)
    with torch.cuda.stream(stream):
        for i in range(max(args.warmup, 3)):
            run(i)
        code = abi.check_status(stream)
        if code != abi.MLA_OK:
            raise RuntimeError(f"device status after warm-up: {abi.status_name(code)}")

        graphs = None
        if not args.no_graph:
            graphs = []
            for i in range(replicas):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=stream):
                    run(i)
                graphs.append(g)
            for i in range(replicas):
                graphs[i].replay()
        torch.cuda.synchronize(dev)

        def one(i):
            if graphs is not None:
                graphs[i % replicas].replay()
            else:
                run(i)

        # ---- timed region: exactly K steps
        clocks = ClockSampler(local)
        clocks.start()
        barrier(world)
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(args.steps):
            one(i)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        barrier(world)
        elapsed_ms = e0.elapsed_time(e1)
        # the spread of single steps, from a second pass of K steps with an
        # event between consecutive ones (kept out of the region above)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
        ev[0].record(stream)
        for i in range(args.steps):
            one(i)
            ev[i + 1].record(stream)
        torch.cuda.synchronize(dev)
        step_ms = sorted(ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps))
        # keep the GPU loaded for at least ~1.5 s so the clock samples cover a busy GPU
        t_end = time.time() + max(0.0, 1.5 - elapsed_ms / 1e3)
        i = args.steps
        while time.time() < t_end:
            one(i)
            i += 1
            if i % 64 == 0:
                torch.cuda.synchronize(dev)
        torch.cuda.synchronize(dev)
        clocks.stop()
        code = abi.check_status(stream)
        if code != abi.MLA_OK:
            raise RuntimeError(f"device status after timing: {abi.status_name(code)}")

        # ---- the attention kernel alone: a CUDA graph of back-to-back launches
        # over the replicas (no host time between them), timed with events on
        # the stream it replays on
        attn_avg_ms = time_attention(dws, steps, S, stream, dev, args.steps)
        long_roof = None
        if shape.name != LONG_WORKLOAD and not args.no_long:
            long_roof = measure_long_attention(args, rank, stream, dev, l2)

        proj = measure_projection(args, w, dws, stream, dev, l2, peaks=load_peaks())
        accept = measure_acceptance(args, stream, dev, l2, peaks=load_peaks())
        gqa = measure_gqa(args, w, dws, steps, stream, dev, l2, peaks=load_peaks())
        e2e_fwd = measure_e2e_forward(args, w, stream, dev)

        # ---- end to end through the public API with host buffers: the step's
        # inputs (queries, new entries, lengths, positions) packed in one pinned
        # host buffer, copied in one transfer to a device buffer whose views the
        # step reads; the step's output read back in one transfer
        names = ("q_nope", "q_pe", "c_new", "kr_new", "kv_len", "start_pos")
        layout, off = [], 0
        for k in names:
            t = getattr(w, k)
            nbytes = t.numel() * t.element_size()
            layout.append((k, off, t.dtype, tuple(t.shape), nbytes))
            off = (off + nbytes + 255) // 256 * 256
        host_pack = torch.empty(off, dtype=torch.uint8).pin_memory()
        for k, o, dt, sh, nb in layout:
            host_pack[o:o + nb].copy_(getattr(w, k).contiguous().view(-1).view(torch.uint8))
        dev_packs = [torch.empty(off, dtype=torch.uint8, device=dev) for _ in range(replicas)]
        views = [{k: dp[o:o + nb].view(dt).view(sh) for k, o, dt, sh, nb in layout} for dp in dev_packs]
        out_dev = steps[0].out if steps[0].out is not None else steps[0].o
        host_out = torch.empty(out_dev.shape, dtype=out_dev.dtype).pin_memory()
        h2d = off
        d2h = host_out.numel() * host_out.element_size()

        # Pipelined like a serving loop: a second stream uploads step i + 1's
        # inputs and reads back step i's output while step i computes; every
        # step still moves its own bytes inside the timed region.  Replica r's
        # device inputs and output are reused by step i + replicas only after
        # step i's compute and read-back have completed.
        copy_stream = torch.cuda.Stream(dev)
        host_outs = [torch.empty(out_dev.shape, dtype=out_dev.dtype).pin_memory() for _ in range(replicas)]
        ev = lambda: torch.cuda.Event()  # noqa: E731
        h2d_done = [ev() for _ in range(replicas)]
        comp_done = [ev() for _ in range(replicas)]
        d2h_done = [ev() for _ in range(replicas)]
        used = [False] * replicas

        def upload(i):
            r = i % replicas
            if used[r]:
                copy_stream.wait_event(comp_done[r])  # step i - replicas has read its inputs
            with torch.cuda.stream(copy_stream):
                dev_packs[r].copy_(host_pack, non_blocking=True)
            h2d_done[r].record(copy_stream)

        def e2e_run(n):
            upload(0)
            for i in range(n):
                r = i % replicas
                if i + 1 < n:
                    upload(i + 1)
                d, st, v = dws[r], steps[r], views[r]
                stream.wait_event(h2d_done[r])
                if used[r]:
                    stream.wait_event(d2h_done[r])  # step i - replicas's output has been read back
                res = st(v["q_nope"], v["q_pe"], v["kv_len"], d.w_uk, d.w_uv, d.w_o, c_new=v["c_new"],
                         kr_new=v["kr_new"], start_pos=v["start_pos"])
                comp_done[r].record(stream)
                used[r] = True
                copy_stream.wait_event(comp_done[r])
                with torch.cuda.stream(copy_stream):
                    host_outs[r].copy_(res, non_blocking=True)
                d2h_done[r].record(copy_stream)
            stream.wait_stream(copy_stream)

        def e2e_step_serial(i):
            r = i % replicas
            d, st, v = dws[r], steps[r], views[r]
            dev_packs[r].copy_(host_pack, non_blocking=True)
            res = st(v["q_nope"], v["q_pe"], v["kv_len"], d.w_uk, d.w_uv, d.w_o, c_new=v["c_new"],
                     kr_new=v["kr_new"], start_pos=v["start_pos"])
            host_outs[r].copy_(res, non_blocking=True)

        def e2e_run_serial(n):
            for i in range(n):
                e2e_step_serial(i)

        # The loop that is faster on this machine is timed: the pipelined one
        # hides the copies behind the compute but makes more host calls per
        # step (a second stream, its events), which a short step cannot hide
        # (on the GB300 machine: ~80 us of host time per step against ~50 us for
        # the loop with the copies in line on the step's stream).
        # the step replays as a CUDA graph captured through the public API
        # (DecodeStep(graph=True)) unless --no-graph: one launch per step.
        # Each replica's graph is captured here, on its filled input buffers,
        # so that no capture falls in a trial or the timed region.
        for r, st in enumerate(steps):
            st.graph = graphs is not None
            if st.graph:
                d, v = dws[r], views[r]
                dev_packs[r].copy_(host_pack)
                st(v["q_nope"], v["q_pe"], v["kv_len"], d.w_uk, d.w_uv, d.w_o, c_new=v["c_new"], kr_new=v["kr_new"],
                   start_pos=v["start_pos"])
        torch.cuda.synchronize(dev)

        def trial(fn, n=32):
            fn(2)
            torch.cuda.synchronize(dev)
            t0 = time.perf_counter()
            fn(n)
            torch.cuda.synchronize(dev)
            return time.perf_counter() - t0

        # best of three short runs each (host timing jitter decides otherwise)
        pipelined = min(trial(e2e_run) for _ in range(3)) <= min(trial(e2e_run_serial) for _ in range(3))
        run = e2e_run if pipelined else e2e_run_serial
        run(3)
        torch.cuda.synchronize(dev)
        barrier(world)
        x0, x1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        x0.record(stream)
        copy_stream.wait_stream(stream)  # the first upload starts after x0
        run(args.steps)
        x1.record(stream)  # after the last read-back (the stream waited on the copy stream)
        torch.cuda.synchronize(dev)
        e2e_ms = x0.elapsed_time(x1)
        assert abi.check_status(stream) == abi.MLA_OK

    max_ms = max_over_ranks(elapsed_ms, world, dev)
    max_e2e = max_over_ranks(e2e_ms, world, dev)
    total_bytes = sum_over_ranks(float(cache_bytes) * args.steps, world, dev)
    ms_step = max_ms / args.steps
    peaks = load_peaks()
    roof = attention_roofline(w, attn_avg_ms, peaks)

    def pct(q):
        return round(step_ms[min(len(step_ms) - 1, int(q * len(step_ms)))] * 1e3, 3)
    launches_per_step = 1 + 1 + 1 + 1 + (2 if shape.hidden else 1)  # append, absorb, attention, combine, W_UV (+ W_O)
    line = {
        "metric": METRIC,
        "value": round(total_bytes / (max_ms * 1e-3) / 1e9, 2),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_step, 6),
        "us_per_step": round(ms_step * 1e3, 3),
        "attn_us_per_launch": round(attn_avg_ms * 1e3, 3),
        "attn_combine_us": gqa.get("mla_us") if isinstance(gqa, dict) else None,
        "queries_per_s": round(world * shape.batch * shape.q_len / (ms_step * 1e-3), 1),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) caches and queries, N(0,1/sqrt(fan_in)) weights)",
        "config": {
            "workload": shape.name, "batch": shape.batch, "q_len": shape.q_len, "heads": shape.num_heads,
            "kv_groups": shape.num_kv_groups, "rank": shape.rank, "d_rope": shape.d_rope, "d_nope": shape.d_nope,
            "d_v": shape.d_v, "hidden": shape.hidden,
            "kv_len": (shape.kv_lo if shape.kv_lo == shape.kv_hi else [shape.kv_lo, shape.kv_hi]),
            "layout": "paged(64)" if shape.paged else "contiguous", "num_splits": S,
            "cache_bytes_per_step": cache_bytes,
            "l2": f"inputs rotate over {replicas} replicas of {per_replica / 2**20:.1f} MiB (> 2x L2 of "
                  f"{l2 / 2**20:.0f} MiB); no flush",
            "cuda_graph": graphs is not None, "parallelism": f"replicas{world}",
        },
        "roofline": roof,
        "roofline_long": long_roof,
        "step_us_dist": {"p10": pct(0.1), "p50": pct(0.5), "p90": pct(0.9)},
        "clocks": clocks.summary(),
        "e2e": {"value": round(total_bytes / (max_e2e * 1e-3) / 1e9, 2), "unit": "GB/s", "pipelined": pipelined,
                "graph": graphs is not None,
                "us_per_step": round(max_e2e / args.steps * 1e3, 3),
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": launches_per_step * args.steps,
        "project_append": proj,
        "acceptance_stats": accept,
        "gqa_comparison": gqa,
        "e2e_loss_forward": e2e_fwd,
    }
    return line, w


def time_attention(dws, steps, S, stream, dev, n_steps):
    """Mean time (ms) of one attention launch (mla_decode_attn): a CUDA graph
    of back-to-back launches over the replicas, timed with CUDA events on the
    stream the graph replays on."""
    import torch
    from paper_2607_27269_gb300 import abi

    replicas = len(dws)
    n_attn = max(replicas, min(max(n_steps, 16), 4 * replicas))
    g_attn = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_attn, stream=stream):
        for i in range(n_attn):
            d, st = dws[i % replicas], steps[i % replicas]
            abi.decode_attn(d.dims, d.cache, d.kv_len, d.max_kv_len, st.q_abs, st.o_part, st.lse_part, S, stream)
    for _ in range(2):
        g_attn.replay()
    torch.cuda.synchronize(dev)
    marks = []
    for _ in range(max(3, n_steps // n_attn)):
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        g_attn.replay()
        a1.record(stream)
        marks.append((a0, a1))
    torch.cuda.synchronize(dev)
    code = abi.check_status(stream)
    if code != abi.MLA_OK:
        raise RuntimeError(f"device status after the attention launches: {abi.status_name(code)}")
    ms = [a.elapsed_time(b) / n_attn for a, b in marks]
    return sum(ms) / len(ms)


def attention_roofline(w, attn_ms, peaks):
    """Roofline of the attention core on workload `w` from its mean launch
    time: algorithmic bytes = the latent + positional cache read once for all
    heads; algorithmic FLOPs = scores over the visible keys plus P C."""
    shape = w.shape
    cache_bytes = w.cache_bytes
    achieved = cache_bytes / (attn_ms * 1e-3) / 1e9
    # per query (b, i, head) with kv_b - q + i + 1 visible keys: 2 (r + d_rope)
    # per key for the scores and 2 r for P C
    kv = [int(x) for x in w.kv_len.tolist()]
    keys = sum(k - shape.q_len + i + 1 for k in kv for i in range(shape.q_len)) * shape.num_heads
    flops = float(keys) * (2 * (shape.rank + shape.d_rope) + 2 * shape.rank)
    tflops = flops / (attn_ms * 1e-3) / 1e12
    t_floor = max(cache_bytes / (peaks["hbm_gbs"] * 1e9), flops / (peaks["bf16_tflops"] * 1e12))
    return {
        "bound": "hbm", "achieved": round(achieved, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
        "frac": round(achieved / peaks["hbm_gbs"], 4), "traffic": attn_traffic(shape.name),
        "peak_source": peaks["source"], "kernel": "mla_decode_attn", "workload": shape.name,
        "bytes_per_launch": cache_bytes, "attn_us_per_launch": round(attn_ms * 1e3, 3),
        "flops_per_launch": flops, "achieved_tflops": round(tflops, 1),
        "tensor_frac": round(tflops / peaks["bf16_tflops"], 4),
        "ridge_frac": round(t_floor / (attn_ms * 1e-3), 4),
        "nominal_gbs": NOMINAL_HBM_GBS, "nominal_frac": round(achieved / NOMINAL_HBM_GBS, 4),
    }


def measure_long_attention(args, rank, stream, dev, l2):
    """The attention core on the long-context workload, rated like the main
    one (replicas beyond 2x L2, a CUDA graph of back-to-back launches)."""
    import torch
    from paper_2607_27269_gb300 import abi
    from paper_2607_27269_gb300 import workloads as wl

    w = wl.make(wl.SHAPES[LONG_WORKLOAD], seed=args.seed + rank)
    per = (w.c_kv.numel() + w.k_rope.numel()) * 2
    replicas = max(2, math.ceil(2 * l2 / per) + 1)
    dws = [abi.to_device(w, dev) for _ in range(replicas)]
    steps = [abi.DecodeStep(d.dims, d.cache, d.batch, d.q_len, d.max_kv_len, args.num_splits) for d in dws]
    for d, st in zip(dws, steps):  # the appended entries and the absorbed queries the attention reads
        st(d.q_nope, d.q_pe, d.kv_len, d.w_uk, d.w_uv, d.w_o, c_new=d.c_new, kr_new=d.kr_new, start_pos=d.start_pos,
           stream=stream)
    torch.cuda.synchronize(dev)
    ms = time_attention(dws, steps, steps[0].num_splits, stream, dev, args.steps)
    roof = attention_roofline(w, ms, load_peaks())
    roof["num_splits"] = steps[0].num_splits
    roof["replicas"] = replicas
    del dws, steps
    torch.cuda.empty_cache()
    return roof


def measure_e2e_forward(args, w, stream, dev):
    """One forward of the E2E functional-reconstruction loss (Sec. 4.1) on the
    workload's new tokens: the converted MLA layer from hidden states and the
    original GQA layer on the same states, the shared W_O, the masked MSE.
    Timed as a CUDA graph of back-to-back forwards on one copy (the caches stay
    resident; the new entries are rewritten in place each time)."""
    import torch
    from paper_2607_27269_gb300 import abi
    from paper_2607_27269_gb300 import workloads as wl

    s = w.shape
    p = wl.projection(w, seed=args.seed)
    gw = wl.gqa(w, seed=args.seed)
    gp = wl.gqa_projection(w, seed=args.seed)
    if w.w_o is None:
        return {"skipped": "no output projection at this shape"}
    dw = abi.to_device(w, dev)
    step = abi.DecodeStep(dw.dims, dw.cache, dw.batch, dw.q_len, dw.max_kv_len)
    gdims = abi.GqaDims(gw.num_heads, gw.num_kv_groups, gw.d, gw.sm_scale, s.rope_style, s.rope_base)
    bt = None if gw.block_table is None else gw.block_table.to(dev)
    gcache = abi.Cache(gw.v_cache.to(dev), gw.k_cache.to(dev), gw.capacity, bt, s.page_size if s.paged else 0,
                       gw.num_pages)
    fwd = abi.E2EForward(step, gdims, gcache, p.hidden)
    mla_w = tuple(t.to(dev) for t in (p.w_dkv, p.w_kr, p.w_q, w.w_uk, w.w_uv))
    gqa_w = tuple(t.to(dev) for t in (gp.w_q, gp.w_k, gp.w_v))
    h, w_o = p.h.to(dev), w.w_o.to(dev)
    us = _graph_time_us(lambda i: fwd(h, mla_w, gqa_w, w_o, dw.start_pos, dw.kv_len, stream=stream), 16, stream, dev)
    code = abi.check_status(stream)
    if code != abi.MLA_OK:
        raise RuntimeError(f"device status after the E2E forward: {abi.status_name(code)}")
    return {"us_per_forward": round(us, 3), "tokens": int(w.kv_len.numel() * s.q_len), "hidden": p.hidden,
            "loss": round(float(fwd.loss.item()), 6)}


def _graph_time_us(launch, n_launch, stream, dev):
    import torch
    for i in range(3):
        launch(i)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(n_launch):
            launch(i)
    g.replay()
    torch.cuda.synchronize(dev)
    times = []
    for _ in range(5):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        g.replay()
        b.record(stream)
        times.append((a, b))
    torch.cuda.synchronize(dev)
    return sum(a.elapsed_time(b) for a, b in times) / len(times) / n_launch * 1e3


def measure_gqa(args, w, dws, steps, stream, dev, l2, peaks):
    """The original GQA draft's attention at the same shape (mla_gqa_decode_attn:
    split-KV attention and merge) beside the MLA path's (mla_decode_attn +
    mla_combine), both as CUDA graphs of back-to-back calls over replicas
    beyond 2x L2.  Bytes: the cache each reads per step."""
    import torch
    from paper_2607_27269_gb300 import abi
    from paper_2607_27269_gb300 import workloads as wl

    gw = wl.gqa(w, seed=args.seed)
    s = w.shape
    per = (gw.k_cache.numel() + gw.v_cache.numel()) * 2
    reps = max(2, math.ceil(2 * l2 / per) + 1)
    dims = abi.GqaDims(gw.num_heads, gw.num_kv_groups, gw.d, gw.sm_scale, s.rope_style, s.rope_base)
    runs = []
    for _ in range(reps):
        bt = None if gw.block_table is None else gw.block_table.to(dev)
        cache = abi.Cache(gw.v_cache.to(dev), gw.k_cache.to(dev), gw.capacity, bt, s.page_size if s.paged else 0,
                          gw.num_pages)
        st = abi.GqaStep(dims, cache, gw.kv_len.numel(), gw.q.shape[1], int(gw.kv_len.max()), args.num_splits)
        runs.append((st, gw.q.to(dev), gw.kv_len.to(dev)))
    n = max(reps, 16)
    gqa_us = _graph_time_us(lambda i: runs[i % reps][0](runs[i % reps][1], runs[i % reps][2], stream=stream), n,
                            stream, dev)
    code = abi.check_status(stream)
    if code != abi.MLA_OK:
        raise RuntimeError(f"device status after the GQA attention: {abi.status_name(code)}")
    R = len(dws)

    def mla(i):
        d, st = dws[i % R], steps[i % R]
        abi.decode_attn(d.dims, d.cache, d.kv_len, d.max_kv_len, st.q_abs, st.o_part, st.lse_part, st.num_splits,
                        stream)
        abi.combine(d.dims, d.batch, d.q_len, d.kv_len, d.max_kv_len, st.o_part, st.lse_part, st.o_lat, st.lse,
                    st.num_splits, stream)

    mla_us = _graph_time_us(mla, max(R, 16), stream, dev)
    gqa_bytes, mla_bytes = gw.cache_bytes, w.cache_bytes
    gbs = gqa_bytes / (gqa_us * 1e-6) / 1e9
    del runs
    return {"kernel": "mla_gqa_decode_attn", "head_dim": gw.d, "gqa_us": round(gqa_us, 3),
            "mla_us": round(mla_us, 3), "gqa_cache_bytes": gqa_bytes, "mla_cache_bytes": mla_bytes,
            "cache_bytes_ratio_mla_over_gqa": round(mla_bytes / gqa_bytes, 4),
            "time_ratio_mla_over_gqa": round(mla_us / gqa_us, 4), "gqa_achieved_gbs": round(gbs, 1),
            "gqa_frac": round(gbs / peaks["hbm_gbs"], 4), "replicas": reps, "peak_source": peaks["source"]}


def measure_acceptance(args, stream, dev, l2, peaks):
    """Acceptance statistics (mla_acceptance_stats) of draft against target
    logits for every (sequence, query position) of the workload, over the
    vocabulary of the model the shape follows, timed alone: a CUDA graph of
    back-to-back launches over enough logits replicas that the bytes between
    two reuses exceed 2x L2.  Algorithmic bytes: one read of both logits."""
    import torch
    from paper_2607_27269_gb300 import abi
    from paper_2607_27269_gb300 import workloads as wl

    lg = wl.logits(args.workload, seed=args.seed)
    rows, vocab = lg.draft.shape
    nbytes = 2 * lg.draft.numel() * lg.draft.element_size()
    reps = max(2, math.ceil(2 * l2 / nbytes) + 1)
    pairs = [(lg.draft.to(dev), lg.target.to(dev)) for _ in range(reps)]
    outs = [torch.empty(rows, dtype=torch.float32, device=dev)] + [
        torch.empty(rows, dtype=torch.int32, device=dev) for _ in range(3)]
    n_launch = max(reps, 16)

    def launch(i):
        d, t = pairs[i % reps]
        abi.acceptance_stats(d, t, *outs, stream=stream)

    for i in range(3):
        launch(i)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(n_launch):
            launch(i)
    g.replay()
    torch.cuda.synchronize(dev)
    times = []
    for _ in range(5):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        g.replay()
        b.record(stream)
        times.append((a, b))
    torch.cuda.synchronize(dev)
    us = sum(a.elapsed_time(b) for a, b in times) / len(times) / n_launch * 1e3
    gbs = nbytes / (us * 1e-6) / 1e9
    return {"kernel": "mla_acceptance_stats", "us_per_launch": round(us, 3), "rows": rows, "vocab": vocab,
            "dtype": "bf16", "bytes_per_launch": nbytes, "achieved_gbs": round(gbs, 1), "bound": "hbm",
            "frac": round(gbs / peaks["hbm_gbs"], 4), "replicas": reps, "peak_source": peaks["source"],
            "mean_alpha_sample": round(float(outs[0].float().mean()), 4)}


def measure_projection(args, w, dws, stream, dev, l2, peaks):
    """The projection that precedes the step (mla_project_append) timed alone:
    a CUDA graph of back-to-back launches over enough weight replicas that
    the weights streamed between two reuses exceed 2x L2.  Reported beside
    the step (it is not part of the step's bytes)."""
    import torch
    from paper_2607_27269_gb300 import abi
    from paper_2607_27269_gb300 import workloads as wl

    s = w.shape
    p = wl.projection(w, seed=args.seed)
    D = p.hidden
    B, n = w.c_new.shape[0], w.c_new.shape[1]
    M = B * n
    nq = s.num_heads * (s.d_nope + s.d_rope)
    weight_bytes = (s.rank + s.d_rope + nq) * D * 2
    io_bytes = M * D * 2 + M * (s.rank + s.d_rope + nq) * 2
    flops = 2.0 * M * D * (s.rank + s.d_rope + nq)
    reps = max(2, math.ceil(2 * l2 / weight_bytes) + 1)
    dims = abi.Dims(s.num_heads, s.num_kv_groups, s.d_nope, s.d_rope, s.d_v, s.rank, D, s.sm_scale, s.rope_style,
                    s.rope_base)
    h = p.h.to(dev)
    ws = [(p.w_dkv.to(dev), p.w_kr.to(dev), p.w_q.to(dev)) for _ in range(reps)]
    q_nope = torch.empty(B, n, s.num_heads, s.d_nope, dtype=torch.bfloat16, device=dev)
    q_pe = torch.empty(B, n, s.num_heads, s.d_rope, dtype=torch.bfloat16, device=dev)
    n_launch = max(reps, 32)

    def launch(i):
        d = dws[i % len(dws)]
        w_dkv, w_kr, w_q = ws[i % reps]
        abi.project_append(dims, d.cache, h, w_dkv, w_kr, w_q, d.start_pos, q_nope, q_pe, stream)

    for i in range(3):
        launch(i)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(n_launch):
            launch(i)
    g.replay()
    torch.cuda.synchronize(dev)
    times = []
    for _ in range(5):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        g.replay()
        b.record(stream)
        times.append((a, b))
    torch.cuda.synchronize(dev)
    code = abi.check_status(stream)
    if code != abi.MLA_OK:
        raise RuntimeError(f"device status after the projection: {abi.status_name(code)}")
    us = sum(a.elapsed_time(b) for a, b in times) / len(times) / n_launch * 1e3
    gbs = (weight_bytes + io_bytes) / (us * 1e-6) / 1e9
    tflops = flops / (us * 1e-6) / 1e12
    # the bound is whichever roofline time is longer at the measured peaks
    t_hbm = (weight_bytes + io_bytes) / (peaks["hbm_gbs"] * 1e9)
    t_tc = flops / (peaks["bf16_tflops"] * 1e12)
    bound = "tensor" if t_tc > t_hbm else "hbm"
    frac = (tflops / peaks["bf16_tflops"]) if bound == "tensor" else (gbs / peaks["hbm_gbs"])
    return {"kernel": "mla_project_append", "us_per_launch": round(us, 3), "rows": M, "hidden": D,
            "columns": s.rank + s.d_rope + nq, "bytes_per_launch": weight_bytes + io_bytes,
            "flops_per_launch": flops, "achieved_gbs": round(gbs, 1), "achieved_tflops": round(tflops, 2),
            "bound": bound, "frac": round(frac, 4), "weight_replicas": reps, "peak_source": peaks["source"]}


# DRAM bytes (read + write) per attention launch from one ncu capture of the
# kernel source with this sha256 prefix (profiles/attn_tc_<workload>.md); a
# kernel that has changed since reports null.
TRAFFIC_SOURCE = "f5772acba64d9795"
TRAFFIC = {
    "qwen05b_b16_h14_r256_t2048": 21206016,  # at 128 partitions
    "llama3b_long_b8_h24_r512_t16k_32k": 210286592,
    "llama1b_paged_b128_h32_r512_t128_8192": 710535424,
    "llama1b_chunk5_b32_h32_r512_t4096": 164428288,
}


def attn_traffic(workload: str):
    import hashlib
    path = os.path.join(ROOT, "paper_2607_27269_gb300", "csrc", "attn_tc.cu")
    with open(path, "rb") as f:
        h = hashlib.sha256(f.read()).hexdigest()[:16]
    return TRAFFIC.get(workload) if h == TRAFFIC_SOURCE else None


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": p["hbm_gbs"], "bf16_tflops": p["bf16_tflops"], "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "source": "fallback"}


def run_kernel_only(args, local):
    """Profiling aid (for ncu captures of one kernel on one copy of the
    workload): `--proj-launches` launches of the projection or
    `--accept-launches` launches of the acceptance statistics, alone.  Prints
    one JSON line with the device status."""
    import torch
    from paper_2607_27269_gb300 import abi
    from paper_2607_27269_gb300 import workloads as wl

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = wl.make(wl.SHAPES[args.workload], seed=args.seed)
    if args.proj_launches > 0:
        s = w.shape
        p = wl.projection(w, seed=args.seed)
        dw = abi.to_device(w, dev)
        dims = abi.Dims(s.num_heads, s.num_kv_groups, s.d_nope, s.d_rope, s.d_v, s.rank, p.hidden, s.sm_scale,
                        s.rope_style, s.rope_base)
        h, a, b, c = p.h.to(dev), p.w_dkv.to(dev), p.w_kr.to(dev), p.w_q.to(dev)
        qn, qp = torch.empty_like(dw.q_nope), torch.empty_like(dw.q_pe)
        for _ in range(args.proj_launches):
            abi.project_append(dims, dw.cache, h, a, b, c, dw.start_pos, qn, qp)
        kind, n = "project_append_only", args.proj_launches
    elif args.gqa_launches > 0:
        s = w.shape
        gw = wl.gqa(w, seed=args.seed)
        dims = abi.GqaDims(gw.num_heads, gw.num_kv_groups, gw.d, gw.sm_scale, s.rope_style, s.rope_base)
        bt = None if gw.block_table is None else gw.block_table.to(dev)
        cache = abi.Cache(gw.v_cache.to(dev), gw.k_cache.to(dev), gw.capacity, bt, s.page_size if s.paged else 0,
                          gw.num_pages)
        st = abi.GqaStep(dims, cache, gw.kv_len.numel(), gw.q.shape[1], int(gw.kv_len.max()), args.num_splits)
        q, kv = gw.q.to(dev), gw.kv_len.to(dev)
        for _ in range(args.gqa_launches):
            st(q, kv)
        kind, n = "gqa_attention_only", args.gqa_launches
    else:
        lg = wl.logits(args.workload, seed=args.seed)
        d, t = lg.draft.to(dev), lg.target.to(dev)
        for _ in range(args.accept_launches):
            abi.acceptance_stats(d, t)
        kind, n = "acceptance_only", args.accept_launches
    torch.cuda.synchronize(dev)
    code = abi.check_status()
    return {"profile": kind, "workload": w.shape.name, "launches": n, "status": abi.status_name(code)}, code


def run_attn_only(args, local):
    """Profiling aid (for ncu captures of one kernel on one copy of the
    workload): one full decode step, then `--attn-launches` launches of the
    attention kernel alone.  Prints one JSON line with the device status."""
    import torch
    from paper_2607_27269_gb300 import abi
    from paper_2607_27269_gb300 import workloads as wl

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = wl.make(wl.SHAPES[args.workload], seed=args.seed)
    d = abi.to_device(w, dev)
    st = abi.DecodeStep(d.dims, d.cache, d.batch, d.q_len, d.max_kv_len, args.num_splits)
    st(d.q_nope, d.q_pe, d.kv_len, d.w_uk, d.w_uv, d.w_o, c_new=d.c_new, kr_new=d.kr_new, start_pos=d.start_pos)
    for _ in range(args.attn_launches):
        abi.decode_attn(d.dims, d.cache, d.kv_len, d.max_kv_len, st.q_abs, st.o_part, st.lse_part, st.num_splits)
    torch.cuda.synchronize(dev)
    code = abi.check_status()
    return {"profile": "attn_only", "workload": w.shape.name, "launches": args.attn_launches,
            "num_splits": st.num_splits, "cache_bytes": w.cache_bytes, "status": abi.status_name(code)}, code


# ---------------------------------------------------------------- the oracle on the host

def oracle_sample(w, budget_s: float = 20.0):
    """Run the fp64 oracle on growing subsets of the workload's sequences until
    about `budget_s` seconds of CPU work have been measured.  Returns
    (GB/s of cache processed, threads, description)."""
    import numpy as np
    from oracle import oracle as orc
    from tests.helpers import bits, dims_of, oracle_cache

    dims = dims_of(w)
    cache = oracle_cache(w)
    orc.cache_append(dims, cache, bits(w.c_new), bits(w.kr_new), w.start_pos.numpy())
    args = (bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk), bits(w.w_uv),
            None if w.w_o is None else bits(w.w_o))
    order = list(np.argsort(-w.kv_len.numpy()))  # longest first, spread over the length mix
    order = order[::2] + order[1::2]
    orc.mla_decode(dims, cache, *args[:5], args[5], seqs=order[:1])  # warm-up (threads, pages)
    done, spent, nbytes, passes = 0, 0.0, 0, 0
    per_tok = (w.shape.rank + w.shape.d_rope) * 2
    # growing subsets of the sequences; a small workload is repeated whole
    while spent < budget_s:
        if done == len(order):
            done, passes = 0, passes + 1
        take = max(1, min(len(order) - done, 2 ** max(0, int(math.log2(done + 1)))))
        seqs = order[done:done + take]
        t0 = time.perf_counter()
        orc.mla_decode(dims, cache, *args[:5], args[5], seqs=seqs)
        spent += time.perf_counter() - t0
        nbytes += int(w.kv_len.numpy()[seqs].sum()) * per_tok
        done += take
    what = (f"{passes} passes over all {len(order)} sequences and {done} more" if passes
            else f"{done} of {len(order)} sequences")
    desc = f"{what} of {w.shape.name} ({nbytes / 1e6:.1f} MB of cache), fp64 non-absorbed oracle incl. W_O"
    return nbytes / spent / 1e9, orc.num_threads(), desc, spent


def run_reference(args, rank, world):
    """The reference arm: the CPU oracle, timed as it stands on the host cores."""
    from paper_2607_27269_gb300 import workloads as wl
    from oracle import oracle as orc
    from tests.helpers import bits, dims_of, oracle_cache

    if rank != 0:
        return None
    shape = wl.SHAPES[args.workload]
    w = wl.make(shape, seed=args.seed)
    dims = dims_of(w)
    cache = oracle_cache(w)
    orc.cache_append(dims, cache, bits(w.c_new), bits(w.kr_new), w.start_pos.numpy())
    inputs = (bits(w.q_nope), bits(w.q_pe), w.kv_len.numpy(), bits(w.w_uk), bits(w.w_uv),
              None if w.w_o is None else bits(w.w_o))
    # one step = the oracle on a bounded sample of the workload's sequences,
    # sized from one probe so that warm-up + steps stay within about 2 minutes
    import numpy as np
    order = list(np.argsort(-w.kv_len.numpy()))
    t0 = time.perf_counter()
    orc.mla_decode(dims, cache, *inputs[:5], inputs[5], seqs=order[:1])
    one = max(time.perf_counter() - t0, 1e-4)
    budget = 120.0 / max(args.steps + args.warmup, 1)
    n = int(max(1, min(len(order), budget / one)))
    seqs = order[:n]
    per_tok = (shape.rank + shape.d_rope) * 2
    nbytes = int(w.kv_len.numpy()[seqs].sum()) * per_tok
    for _ in range(args.warmup):
        orc.mla_decode(dims, cache, *inputs[:5], inputs[5], seqs=seqs)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        orc.mla_decode(dims, cache, *inputs[:5], inputs[5], seqs=seqs)
    el = time.perf_counter() - t0
    value = nbytes * args.steps / el / 1e9
    sample = f"{n} of {len(order)} sequences of {shape.name} per step, fp64 non-absorbed oracle incl. W_O"
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(el / args.steps * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": shape.name, "sample": sample},
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": orc.num_threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main(argv=None):
    args = parse_args(argv)
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        if args.impl == "reference":
            if rank != 0:
                return 0
            world = 1
        else:
            import torch
            torch.cuda.set_device(local)
            dist.init_process_group("nccl")
    if args.attn_launches > 0:
        line, code = run_attn_only(args, local)
        print(json.dumps(line), flush=True)
        return 0 if code == 0 else 1
    if args.proj_launches > 0 or args.accept_launches > 0 or args.gqa_launches > 0:
        line, code = run_kernel_only(args, local)
        print(json.dumps(line), flush=True)
        return 0 if code == 0 else 1
    if args.impl == "reference":
        line = run_reference(args, rank, world)
        if line is not None:
            print(json.dumps(line), flush=True)
        return 0
    line, w = run_ours(args, rank, world, local)
    if rank == 0:
        if world == 1 and not args.no_cpu_baseline:
            v, cores, desc, spent = oracle_sample(w)
            line["cpu_baseline"] = {"value": round(v, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
                                    "sample": desc, "seconds": round(spent, 2)}
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
