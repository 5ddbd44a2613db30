#!/usr/bin/env python3
"""Benchmark of prefix-reuse prefill on GB300: one step = restore of the
cached prefix KV into the paged pool + append of the new tokens' KV +
causal GQA attention of the new tokens over [prefix ++ new], for one layer
of the Llama-3-70B-shaped workload (8 requests x 8192 cached + 1024 new
tokens, 64 q heads / 8 kv heads, d 128, page size 16).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  `value` is new-token prefill throughput of
the whole step with inputs already in HBM (restore reads a device staging
buffer); `e2e` is the same metric through the C ABI with the step's inputs
copied from pinned host memory (prefix pages, q, new K/V) and the output
copied back inside the timed region.  Under torchrun each rank runs an
independent replica on its own batch (the path has no exchange step).
`--impl reference` times the float64 CPU oracle on the host cores instead.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "new-token prefill tok/s & attn TFLOP/s vs bf16 peak; KV restore GB/s vs HBM"
WORKLOAD = "llama3-70b-layer"


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


def make_workload(name: str, seed: int):
    from paper_2505_23970_gb300 import workloads as wl
    if name == "70b":
        return wl.llama3_70b_layer(seed=seed)
    if name == "8b":
        return wl.llama3_8b_layer(seed=seed)
    if name == "tiny":
        return wl.tiny(seed=seed)
    if name.startswith("mix"):
        return wl.conversation_mix(seed=seed, hit_p=float(name[3:] or 1.0))
    if name == "long":
        return wl.long_document(seed=seed)
    if name == "long-recompute":
        return wl.long_document(seed=seed, recompute=True)
    raise ValueError(name)


# ----------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while running."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.gpu)],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                rows.append((float(f[1]), float(f[2]), float(f[3]), f[5:9]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        # samples under load: power above the idle floor
        pmax = max(r[2] for r in rows)
        load = [r for r in rows if r[2] >= 0.5 * pmax] or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in load for k, v in enumerate(r[3]) if v == "Active"})
        return {"sm_mhz": statistics.median(r[0] for r in load), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(load), "power_w_max": pmax}


# ------------------------------------------------------------- distributed
def dist_setup(n_gpus: int):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl"
        import torch
        if not torch.cuda.is_available():
            backend = "gloo"
        else:
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------ CPU oracle
def oracle_sample(w, seconds: float, rng, pool=None, threads=None):
    """Time the float64 oracle on a bounded sample of one step and
    extrapolate the full step: restore of a block subset, the full append,
    attention of random (b, h, i) rows until `seconds` have passed."""
    import oracle
    threads = threads or os.cpu_count() or 1
    if pool is None:
        pool = w.empty_pool()
    ids = w.prefix_blocks()
    nb = min(ids.size, 256)
    t0 = time.perf_counter()
    if nb:
        oracle.kv_restore(pool, w.host_src()[:nb], ids[:nb])
    t_restore = (time.perf_counter() - t0) * (ids.size / max(nb, 1))
    if nb < ids.size:  # the rest of the image, untimed, so attention reads real keys
        oracle.kv_restore(pool, w.host_src()[nb:], ids[nb:])
    k, v = w.kv_new()
    t0 = time.perf_counter()
    oracle.kv_append(pool, 0, k, v, w.block_table, w.prefix_lens, w.cu_new_lens)
    t_append = time.perf_counter() - t0
    nonempty = np.flatnonzero(w.new_lens > 0)
    rows_done, t_attn = 0, 0.0
    q = w.q()
    batch = max(threads * 4, 16)
    while t_attn < seconds:
        bsel = rng.choice(nonempty, batch)
        rows = np.stack([bsel, rng.integers(0, w.Hq, batch),
                         (rng.random(batch) * w.new_lens[bsel]).astype(np.int64)], 1).astype(np.int32)
        t0 = time.perf_counter()
        oracle.prefix_attn_rows(q, pool, 0, w.block_table, w.prefix_lens, w.cu_new_lens, w.scale,
                                rows, nthreads=threads)
        t_attn += time.perf_counter() - t0
        rows_done += batch
    total_rows = w.T_new * w.Hq
    t_step = t_restore + t_append + t_attn * total_rows / rows_done
    return {"t_step_s": t_step, "rows": rows_done, "restore_blocks": int(nb),
            "threads": threads, "t_attn_s": t_attn, "pool": pool}


def cpu_baseline_entry(w, seconds=12.0, seed=0):
    s = oracle_sample(w, seconds, np.random.default_rng(seed))
    return {"value": w.T_new / s["t_step_s"], "unit": "tok/s", "cores": s["threads"],
            "kind": "oracle",
            "sample": (f"float64 C oracle on {s['threads']} host threads: restore of "
                       f"{s['restore_blocks']} of {w.prefix_blocks().size} blocks, full append, "
                       f"attention of {s['rows']} random (request, head, row) rows of "
                       f"{w.T_new * w.Hq}; step time extrapolated per block / per row")}


def step_input_bytes(w) -> int:
    """Bytes one step reads: q, the new K/V, the restore's staging image and
    the K/V rows the attention reads (the L2 rule of the timing)."""
    restore_payload = int(w.prefix_blocks().size) * w.page_bytes
    return (w.T_new * w.Hq * w.d * 2 + 2 * w.T_new * w.Hkv * w.d * 2 + 2 * restore_payload +
            int(w.total_lens.sum()) * w.Hkv * w.d * 4)


def arm_config(w, world: int) -> dict:
    """The `config` object both arms print for workload w."""
    step_bytes = step_input_bytes(w)
    flush = step_bytes < 2 * 129 * 2**20
    return {"workload": WORKLOAD, "batch": w.B, "prefix_len": int(w.prefix_lens[0]),
            "new_len": int(w.new_lens[0]), "q_heads": w.Hq, "kv_heads": w.Hkv,
            "head_dim": w.d, "page_size": w.ps, "pool_pages": w.num_pages,
            "parallelism": "replicas" if world > 1 else "single",
            "l2": (f"L2 flushed between steps (512 MB write, outside the step events); "
                   f"step reads {step_bytes / 1e6:.0f} MB" if flush else
                   f"inputs larger than L2: step reads {step_bytes / 1e6:.0f} MB"),
            "step": "restore scatter (device staging -> pool) + append + attention"}


def run_reference(args):
    world, rank, _ = dist_setup(args.gpus)
    if rank != 0:
        return
    w = make_workload(args.config, args.seed)
    rng = np.random.default_rng(args.seed)
    pool = None
    per_step = args.ref_step_seconds or max(1.0, min(6.0, 150.0 / max(args.steps + args.warmup, 1)))
    for _ in range(args.warmup):
        s = oracle_sample(w, per_step / 2, rng, pool)
        pool = s["pool"]
    times, walls = [], []
    last = None
    for _ in range(args.steps):
        t0 = time.perf_counter()
        last = oracle_sample(w, per_step, rng, pool)
        walls.append(time.perf_counter() - t0)
        pool = last["pool"]
        times.append(last["t_step_s"])
    t = statistics.mean(times)
    value = w.T_new / t
    # ms_per_step is the measured wall time of one bounded sample step; the
    # throughput `value` is extrapolated from the sample to the full step
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tok/s",
            "estimated": True,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": statistics.mean(walls) * 1e3,
            "full_step_ms_extrapolated": t * 1e3,
            "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": arm_config(w, world),
            "cpu_baseline": {"value": value, "unit": "tok/s", "cores": last["threads"],
                             "kind": "oracle",
                             "sample": f"each step: {last['rows']} random attention rows, "
                                       f"{last['restore_blocks']} restored blocks, full append; "
                                       "extrapolated to the full step"},
            "e2e": {"value": value, "unit": "tok/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
            "gpu_launches": 0}
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------- GPU arm
def traffic_record(kernel: str, workload: str):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current kernel source."""
    import hashlib
    p = os.path.join(ROOT, "profiles", f"{kernel}_{workload}.json")
    src_file = {"attn_tc2": "attn_tc2.cu", "attn_tc": "attn_tc.cu"}.get(kernel, "kv_copy.cu")
    src = os.path.join(ROOT, "paper_2505_23970_gb300", "csrc", src_file)
    if not os.path.exists(p):
        return None
    d = json.load(open(p))
    sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    return d.get("dram_bytes_per_launch") if d.get("src_sha") == sha else None


def run_ours(args):
    import torch

    from paper_2505_23970_gb300 import binding as gcb
    from paper_2505_23970_gb300.harness import DeviceBatch, bf16_tensor

    world, rank, local = dist_setup(args.gpus)
    torch.cuda.set_device(local)
    pk = peaks()
    w = make_workload(args.config, args.seed + rank)
    db = DeviceBatch(w, device=f"cuda:{local}")
    db.stage()
    stream = torch.cuda.current_stream()
    flops = w.attn_flops()
    restore_payload = db.n_blocks * w.page_bytes
    T_new = w.T_new

    def step(ev=None):
        if ev:
            ev[0].record(stream)
        gcb.gc_kv_restore(db.pool.handle, db.staging, db.block_ids, db.n_blocks, stream, None,
                          gcb.GC_RESTORE_SRC_DEVICE)
        if ev:
            ev[1].record(stream)
        db.append(stream)
        if ev:
            ev[2].record(stream)
        db.attn(stream)
        if ev:
            ev[3].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    status = db.check(stream)
    if status != gcb.GC_OK:
        raise RuntimeError(f"device status {gcb.status_name(status)} after warm-up")

    sampler = ClockSampler(local) if not args.profile else None
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    if sampler:
        sampler.start()
        time.sleep(0.3)
    barrier(world)
    torch.cuda.synchronize()
    # inputs the step reads: q, the new K/V, the restore staging image and the
    # pages the attention reads; below twice the 129 MB L2 a 512 MB buffer is
    # written between steps and each step is timed by its own events
    step_bytes = step_input_bytes(w)
    flush = step_bytes < 2 * 129 * 2**20
    flush_buf = torch.empty(512 * 2**20, dtype=torch.uint8, device=db.q.device) if flush else None
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for k in range(args.steps):
        if flush:
            flush_buf.fill_(k & 0xff)
        step(evs[k])
    t_end.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    clocks = sampler.stop() if sampler else None
    if flush:
        ms = sum(e[0].elapsed_time(e[3]) for e in evs) / args.steps
    else:
        ms = t_start.elapsed_time(t_end) / args.steps
    status = db.check(stream)
    if status != gcb.GC_OK:
        raise RuntimeError(f"device status {gcb.status_name(status)} in the timed region")
    restore_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    append_ms = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
    attn_ms = statistics.mean(e[2].elapsed_time(e[3]) for e in evs)
    ms_max = max_over_ranks(ms, world)
    value = world * T_new / (ms_max / 1e3)

    if args.profile:
        if rank == 0:
            print(json.dumps({"profile_run": True, "ms_per_step": ms, "attn_ms": attn_ms}))
        return

    # ---- end to end through the C ABI with host buffers
    e2e = None
    if not args.no_e2e:
        q_h = bf16_tensor(w.q(), pin=True)
        k, v = w.kv_new()
        k_h, v_h = bf16_tensor(k, pin=True), bf16_tensor(v, pin=True)
        out_h = torch.empty(db.out.shape, dtype=torch.bfloat16).pin_memory()
        h2d = q_h.numel() * 2 + k_h.numel() * 2 + v_h.numel() * 2 + restore_payload
        d2h = out_h.numel() * 2

        def e2e_step():
            db.q.copy_(q_h, non_blocking=True)
            db.k_new.copy_(k_h, non_blocking=True)
            db.v_new.copy_(v_h, non_blocking=True)
            gcb.gc_kv_restore(db.pool.handle, db.host_src, db.block_ids, db.n_blocks, stream,
                              db.staging, 0)
            db.append(stream)
            db.attn(stream)
            out_h.copy_(db.out, non_blocking=True)

        def timed_loop(fn, join=None):
            for _ in range(args.warmup):
                fn()
            torch.cuda.synchronize()
            barrier(world)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for k in range(args.steps):
                fn()
            if join is not None:
                stream.wait_stream(join)  # the last output copies are inside the timing
            b.record(stream)
            torch.cuda.synchronize()
            barrier(world)
            return max_over_ranks(a.elapsed_time(b) / args.steps, world)

        serial_ms = timed_loop(e2e_step)

        # Pipelined: two buffer sets; step k+1's host -> device copies and
        # restore run on a side stream while step k's append and attention run,
        # each step's output copied back to its own pinned buffer.
        db2 = DeviceBatch(w, device=f"cuda:{local}", with_restore=True)
        db2.host_src = db.host_src
        dbs = [db, db2]
        outs_h = [out_h, torch.empty_like(out_h).pin_memory()]
        side = torch.cuda.Stream()
        d2h_stream = torch.cuda.Stream()
        loaded = [torch.cuda.Event(), torch.cuda.Event()]
        computed = [torch.cuda.Event(), torch.cuda.Event()]
        done = [torch.cuda.Event(), torch.cuda.Event()]
        count = [0]

        def e2e_pipelined():
            k = count[0]
            count[0] += 1
            cur = dbs[k & 1]
            side.wait_stream(stream) if k == 0 else side.wait_event(done[k & 1])
            with torch.cuda.stream(side):
                cur.q.copy_(q_h, non_blocking=True)
                cur.k_new.copy_(k_h, non_blocking=True)
                cur.v_new.copy_(v_h, non_blocking=True)
                gcb.gc_kv_restore(cur.pool.handle, cur.host_src, cur.block_ids, cur.n_blocks,
                                  side, cur.staging, 0)
            loaded[k & 1].record(side)
            stream.wait_event(loaded[k & 1])
            cur.append(stream)
            cur.attn(stream)
            computed[k & 1].record(stream)
            # the output goes back on its own stream, so the next step's kernels
            # need not wait for it (step k+2 reuses these buffers only after
            # `done`, through the side stream's wait and `loaded`)
            d2h_stream.wait_event(computed[k & 1])
            with torch.cuda.stream(d2h_stream):
                outs_h[k & 1].copy_(cur.out, non_blocking=True)
            done[k & 1].record(d2h_stream)

        e2e_ms = timed_loop(e2e_pipelined, join=d2h_stream)

        # the same pipeline with the 8-bit cache tier: the cached pages come
        # from an INT8 image (made once with gc_kv_save_q8) and are
        # dequantised into the pool, halving the restore's host-link bytes
        chunk8 = gcb.gc_kv_q8_chunk_bytes(db.pool.cfg)
        img8_bytes = db.n_blocks * w.L * 2 * chunk8
        img8_h = torch.empty(img8_bytes, dtype=torch.uint8).pin_memory()
        stg8 = [torch.empty(img8_bytes, dtype=torch.uint8, device=db.q.device) for _ in range(2)]
        gcb.gc_kv_save_q8(db.pool.handle, img8_h, db.block_ids, db.n_blocks, 0, w.L, stream,
                          stg8[0], 0)
        torch.cuda.synchronize()
        count[0] = 0

        def e2e_pipelined_q8():
            k = count[0]
            count[0] += 1
            cur = dbs[k & 1]
            side.wait_stream(stream) if k == 0 else side.wait_event(done[k & 1])
            with torch.cuda.stream(side):
                cur.q.copy_(q_h, non_blocking=True)
                cur.k_new.copy_(k_h, non_blocking=True)
                cur.v_new.copy_(v_h, non_blocking=True)
                gcb.gc_kv_restore_q8(cur.pool.handle, img8_h, cur.block_ids, cur.n_blocks, 0, w.L,
                                     side, stg8[k & 1], 0)
            loaded[k & 1].record(side)
            stream.wait_event(loaded[k & 1])
            cur.append(stream)
            cur.attn(stream)
            computed[k & 1].record(stream)
            d2h_stream.wait_event(computed[k & 1])
            with torch.cuda.stream(d2h_stream):
                outs_h[k & 1].copy_(cur.out, non_blocking=True)
            done[k & 1].record(d2h_stream)

        e2e_q8_ms = timed_loop(e2e_pipelined_q8, join=d2h_stream)
        h2d_q8 = h2d - restore_payload + img8_bytes
        e2e = {"value": world * T_new / (e2e_ms / 1e3), "unit": "tok/s",
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "ms_per_step": e2e_ms, "gpu_launches_per_step": 3,
               "schedule": "two buffer sets: step k+1's host->device copies and restore on a "
                           "side stream and step k-1's output copy on a third stream overlap "
                           "step k's append and attention",
               "serial_value": world * T_new / (serial_ms / 1e3), "serial_ms_per_step": serial_ms,
               "q8_cache_tier": {"value": world * T_new / (e2e_q8_ms / 1e3),
                                 "ms_per_step": e2e_q8_ms, "h2d_bytes_per_step": int(h2d_q8)}}
        ok2 = db2.check(stream) == gcb.GC_OK
        db2.close()
        if not ok2:
            raise RuntimeError("device status after the pipelined end-to-end loop")
        if db.check(stream) != gcb.GC_OK:
            raise RuntimeError("device status after the end-to-end loop")

    # ---- restore of the full 80-layer KV of one 8192-token prefix
    restore80 = ttft80 = decode = configs = attn_q8 = None
    if not args.no_decode and rank == 0:
        decode = bench_decode(args, pk)
    if not args.no_q8_attn and rank == 0:
        attn_q8 = bench_attn_q8(args, pk)
    if not args.no_configs and rank == 0:
        configs = bench_configs(args, pk)
    if not args.no_restore80 and rank == 0:
        image, restore80 = bench_restore80(args, pk)
        ttft80 = bench_ttft80(args, image)
        del image

    attn_tflops = flops / (attn_ms / 1e3) / 1e12
    restore_gbs = 2 * restore_payload / (restore_ms / 1e3) / 1e9
    peak_t = pk["bf16_tflops"]
    line = {
        "metric": METRIC, "value": value, "unit": "tok/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": arm_config(w, world),
        "roofline": {"bound": "tensor", "achieved": attn_tflops, "peak": peak_t,
                     "unit": "TFLOP/s", "frac": attn_tflops / peak_t,
                     "traffic": traffic_record("attn_tc2", WORKLOAD),
                     "kernel": "attn_tc2_kernel", "peak_source": pk["source"] + " burst",
                     "frac_of_sustained": (attn_tflops / pk["bf16_tflops_sustained"]
                                           if pk.get("bf16_tflops_sustained") else None),
                     "flops_per_launch": flops, "ms_per_launch": attn_ms},
        "roofline_restore": restore_roofline(restore_gbs, restore_payload, restore_ms,
                                             restore80, pk),
        "breakdown_ms": {"restore": restore_ms, "append": append_ms, "attention": attn_ms},
        "attn_tflops": attn_tflops, "restore_gbs": restore_gbs,
        "e2e": e2e, "restore_80layer": restore80, "prefill_80layer": ttft80, "decode": decode,
        "configs": configs, "attn_q8": attn_q8,
        "clocks": clocks,
        "gpu_launches": 3 * args.steps,
    }
    if world == 1 and rank == 0 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline_entry(w, seconds=args.cpu_seconds, seed=args.seed)
    if rank == 0:
        print(json.dumps(line), flush=True)


_CUDART = None


def cudart():
    """The CUDA runtime library, for plain cudaMemcpyAsync copies: the host
    link's reference rate is measured with the same call, sizes and stream
    that the library's staged restore and save issue."""
    global _CUDART
    if _CUDART is None:
        import ctypes
        for name in ("libcudart.so", "libcudart.so.13", "/usr/local/cuda/lib64/libcudart.so"):
            try:
                lib = ctypes.CDLL(name)
            except OSError:
                continue
            lib.cudaMemcpyAsync.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t,
                                            ctypes.c_int, ctypes.c_void_p]
            lib.cudaMemcpyAsync.restype = ctypes.c_int
            _CUDART = lib
            break
    return _CUDART


def memcpy_async(dst, src, nbytes: int, kind: int, stream) -> None:
    """One cudaMemcpyAsync (kind 1: host to device, 2: device to host)."""
    lib = cudart()
    if lib is None:
        raise RuntimeError("libcudart not found")
    e = lib.cudaMemcpyAsync(dst.data_ptr(), src.data_ptr(), nbytes, kind, stream.cuda_stream)
    if e != 0:
        raise RuntimeError(f"cudaMemcpyAsync failed ({e})")


def restore_roofline(step_gbs, step_payload, step_ms, restore80, pk):
    """The restore scatter against HBM.  Headline: the 80-layer scatter of
    2.68 GB (10x the L2), whose writes reach DRAM inside its own events.  The
    268 MB launch inside the step is reported beside it: part of its writes
    are still in the 129 MB L2 when it ends, and the next kernel pays for
    their write-back, so its fraction reads high."""
    step = {"achieved": step_gbs,
            "bytes_per_launch": 2 * step_payload, "ms_per_launch": step_ms,
            "traffic": traffic_record("restore_bulk", WORKLOAD),
            "note": "in-step launch (268 MB payload): writes partly still in L2 at its end, "
                    "so no fraction of HBM is given for it"}
    if restore80:
        a = restore80["scatter_bulk_gbs"]
        return {"bound": "hbm", "achieved": a, "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": a / pk["hbm_gbs"], "traffic": None, "kernel": "restore_bulk_kernel",
                "workload": "80-layer image of one 8192-token prefix, 2.68 GB payload "
                            "(read + write bytes counted)",
                "bytes_per_launch": 2 * restore80["payload_bytes"],
                "ms_per_launch": restore80["ms"]["scatter_bulk"], "in_step": step}
    return {"bound": "hbm", "achieved": step_gbs, "peak": pk["hbm_gbs"], "unit": "GB/s",
            "frac": None, "kernel": "restore_bulk_kernel", "in_step": step,
            "note": "no 80-layer scatter measured in this run: the in-step launch's writes are "
                    "partly still in L2 at its end, so no fraction of HBM is given"}


def bench_restore80(args, pk):
    """Restore of the 80-layer KV of one 8192-token prefix (2.68 GB): the
    scatter from a device staging buffer (read + write bytes vs HBM) and the
    whole pinned host -> pool path (payload bytes), next to a plain pinned
    host -> device cudaMemcpyAsync of the same bytes; then the inverse save
    (pool -> device staging gather, pool -> pinned host) beside a plain
    device -> host copy."""
    import torch

    from paper_2505_23970_gb300 import binding as gcb
    from paper_2505_23970_gb300 import workloads as wl
    from paper_2505_23970_gb300.harness import DeviceBatch

    w = wl.llama3_70b_restore_80layer(seed=args.seed)
    db = DeviceBatch(w)
    payload = db.n_blocks * w.page_bytes
    stream = torch.cuda.current_stream()
    reps = 10

    def timed(fn, rounds=1):
        """Mean ms per call over `reps` back-to-back calls; the best of
        `rounds` such runs (the host link's rate varies from run to run)."""
        best = None
        for _ in range(rounds):
            for _ in range(2):
                fn()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(reps):
                fn()
            b.record(stream)
            torch.cuda.synchronize()
            t = a.elapsed_time(b) / reps
            best = t if best is None else min(best, t)
        return best

    db.stage()
    scatter_ms = timed(lambda: gcb.gc_kv_restore(db.pool.handle, db.staging, db.block_ids,
                                                 db.n_blocks, stream, None,
                                                 gcb.GC_RESTORE_SRC_DEVICE))
    vec_ms = timed(lambda: gcb.gc_kv_restore(db.pool.handle, db.staging, db.block_ids,
                                             db.n_blocks, stream, None,
                                             gcb.GC_RESTORE_SRC_DEVICE | gcb.GC_RESTORE_VECTOR))
    # host-link legs, each the best of 3 runs: the staged restore (one
    # cudaMemcpyAsync of the image + the scatter), the zero-copy restore, and
    # the reference rate of the link itself: the same cudaMemcpyAsync of the
    # same bytes on the same stream, with nothing else
    staged_ms = timed(lambda: gcb.gc_kv_restore(db.pool.handle, db.host_src, db.block_ids,
                                                db.n_blocks, stream, db.staging, 0), rounds=3)
    zc_ms = timed(lambda: gcb.gc_kv_restore(db.pool.handle, db.host_src, db.block_ids,
                                            db.n_blocks, stream, None, 0), rounds=3)
    h2d_ms = timed(lambda: memcpy_async(db.staging, db.host_src, payload, 1, stream), rounds=3)
    h2d_torch_ms = timed(lambda: db.staging.copy_(db.host_src, non_blocking=True))
    # the inverse path: save the same pages back to the cache tier
    host_dst = torch.empty_like(db.host_src).pin_memory()
    save_dev_ms = timed(lambda: gcb.gc_kv_save(db.pool.handle, db.staging, db.block_ids,
                                               db.n_blocks, stream, None,
                                               gcb.GC_SAVE_DST_DEVICE))
    save_staged_ms = timed(lambda: gcb.gc_kv_save(db.pool.handle, host_dst, db.block_ids,
                                                  db.n_blocks, stream, db.staging, 0), rounds=3)
    save_zc_ms = timed(lambda: gcb.gc_kv_save(db.pool.handle, host_dst, db.block_ids,
                                              db.n_blocks, stream, None, 0), rounds=3)
    d2h_ms = timed(lambda: memcpy_async(host_dst, db.staging, payload, 2, stream), rounds=3)
    del host_dst
    # the 8-bit cache tier: INT8 image of the same pages
    n, L = db.n_blocks, w.L
    q8_bytes = n * L * 2 * gcb.gc_kv_q8_chunk_bytes(db.pool.cfg)
    q8_dev = torch.empty(q8_bytes, dtype=torch.uint8, device=db.staging.device)
    q8_stg = torch.empty_like(q8_dev)
    q8_host = torch.empty(q8_bytes, dtype=torch.uint8).pin_memory()
    q8_save_ms = timed(lambda: gcb.gc_kv_save_q8(db.pool.handle, q8_dev, db.block_ids, n, 0, L,
                                                 stream, None, gcb.GC_SAVE_DST_DEVICE))
    q8_restore_ms = timed(lambda: gcb.gc_kv_restore_q8(db.pool.handle, q8_dev, db.block_ids, n, 0,
                                                       L, stream, None,
                                                       gcb.GC_RESTORE_SRC_DEVICE))
    q8_save_host_ms = timed(lambda: gcb.gc_kv_save_q8(db.pool.handle, q8_host, db.block_ids, n, 0,
                                                      L, stream, q8_stg, 0))
    q8_staged_ms = timed(lambda: gcb.gc_kv_restore_q8(db.pool.handle, q8_host, db.block_ids, n, 0,
                                                      L, stream, q8_stg, 0))
    q8_zc_ms = timed(lambda: gcb.gc_kv_restore_q8(db.pool.handle, q8_host, db.block_ids, n, 0, L,
                                                  stream, None, 0))
    del q8_dev, q8_stg, q8_host
    ok = db.check(stream) == gcb.GC_OK
    db.close()
    gbs = lambda nbytes, ms: nbytes / (ms / 1e3) / 1e9  # noqa: E731
    return w.host_src(), {
        "payload_bytes": payload, "device_status_ok": ok,
        "scatter_bulk_gbs": gbs(2 * payload, scatter_ms),
        "scatter_bulk_frac_hbm": gbs(2 * payload, scatter_ms) / pk["hbm_gbs"],
        "scatter_vector_gbs": gbs(2 * payload, vec_ms),
        "host_to_pool_staged_gbs": gbs(payload, staged_ms),
        "host_to_pool_zero_copy_gbs": gbs(payload, zc_ms),
        "pinned_h2d_memcpy_gbs": gbs(payload, h2d_ms),
        "pinned_h2d_torch_copy_gbs": gbs(payload, h2d_torch_ms),
        # the host path against the link's own rate (the same cudaMemcpyAsync);
        # the staged path adds the scatter, so it stays below 1
        "host_to_pool_staged_frac_link": h2d_ms / staged_ms,
        "host_to_pool_zero_copy_frac_link": h2d_ms / zc_ms,
        "save_gather_gbs": gbs(2 * payload, save_dev_ms),
        "save_gather_frac_hbm": gbs(2 * payload, save_dev_ms) / pk["hbm_gbs"],
        "pool_to_host_staged_gbs": gbs(payload, save_staged_ms),
        "pool_to_host_zero_copy_gbs": gbs(payload, save_zc_ms),
        "pinned_d2h_memcpy_gbs": gbs(payload, d2h_ms),
        "pool_to_host_staged_frac_link": d2h_ms / save_staged_ms,
        "pool_to_host_zero_copy_frac_link": d2h_ms / save_zc_ms,
        "link_reference": "best of 3 runs of 10 cudaMemcpyAsync calls of the whole image on "
                          "the restore's stream, measured next to the restore / save paths",
        "q8": {
            "image_bytes": q8_bytes,
            "dequant_scatter_gbs": gbs(q8_bytes + payload, q8_restore_ms),
            "dequant_scatter_frac_hbm": gbs(q8_bytes + payload, q8_restore_ms) / pk["hbm_gbs"],
            "quant_gather_gbs": gbs(payload + q8_bytes, q8_save_ms),
            "quant_gather_frac_hbm": gbs(payload + q8_bytes, q8_save_ms) / pk["hbm_gbs"],
            "host_to_pool_staged_image_gbs": gbs(q8_bytes, q8_staged_ms),
            "host_to_pool_staged_bf16_equiv_gbs": gbs(payload, q8_staged_ms),
            "host_to_pool_zero_copy_bf16_equiv_gbs": gbs(payload, q8_zc_ms),
            "pool_to_host_staged_image_gbs": gbs(q8_bytes, q8_save_host_ms),
            "ms": {"dequant_scatter": q8_restore_ms, "quant_gather": q8_save_ms,
                   "staged": q8_staged_ms, "zero_copy": q8_zc_ms,
                   "save_staged": q8_save_host_ms},
        },
        "ms": {"scatter_bulk": scatter_ms, "scatter_vector": vec_ms, "staged": staged_ms,
               "zero_copy": zc_ms, "h2d_memcpy": h2d_ms, "h2d_torch_copy": h2d_torch_ms,
               "save_gather": save_dev_ms,
               "save_staged": save_staged_ms, "save_zero_copy": save_zc_ms,
               "d2h_memcpy": d2h_ms},
    }


CONFIG_SET = ("tiny", "8b", "70b", "mix0", "mix0.5", "mix1", "long", "long-recompute")


def bench_configs(args, pk):
    """Every configuration of the workload set, each timed on its own: one
    step = restore scatter (device staging -> pool) + append + attention of
    one layer, plus the same step end to end through the C ABI (inputs from
    pinned host memory, restore staged from the pinned image, output copied
    back, one stream).  Lengths, block tables and pool sizes come from the
    seeded workload definitions; the tensors (q, the new K/V, the cached
    image) are drawn N(0,1) on the device from a seeded torch generator and
    rounded to bf16, since the numpy draws of the larger configs would take
    minutes on the host.  Steps whose inputs are smaller than twice the L2 are
    separated by a 512 MB write and timed by their own events."""
    import torch

    from paper_2505_23970_gb300 import binding as gcb
    from paper_2505_23970_gb300.harness import _i32

    dev = torch.device("cuda", torch.cuda.current_device())
    stream = torch.cuda.current_stream()
    peak_t, peak_h = pk["bf16_tflops"], pk["hbm_gbs"]
    res = {}
    flush_buf = torch.empty(512 * 2**20, dtype=torch.uint8, device=dev)
    # the host link's reference rate: best of 3 pinned 256 MB host -> device
    # cudaMemcpyAsync calls on the bench stream
    link_h = torch.empty(256 * 2**20, dtype=torch.uint8).pin_memory()
    link_d = torch.empty_like(link_h, device=dev)
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    link_ms = []
    for _ in range(3):
        a.record(stream)
        memcpy_async(link_d, link_h, link_h.numel(), 1, stream)
        b.record(stream)
        torch.cuda.synchronize()
        link_ms.append(a.elapsed_time(b))
    link_gbs = link_h.numel() / (min(link_ms) / 1e3) / 1e9
    del link_h, link_d
    for name in CONFIG_SET:
        t_cfg = time.perf_counter()
        w = make_workload(name, args.seed)
        gen = torch.Generator(device=dev)
        gen.manual_seed(1000 + args.seed)

        def randn(*shape):
            return torch.randn(shape, generator=gen, device=dev, dtype=torch.float32).to(
                torch.bfloat16)

        pool = gcb.KVPool.create(w.L, w.Hkv, w.d, w.ps, w.num_pages, device=dev)
        pool.planes().view(torch.int16).fill_(0x7FC0)
        bt, pl, nl, cu = (_i32(w.block_table, dev), _i32(w.prefix_lens, dev),
                          _i32(w.new_lens, dev), _i32(w.cu_new_lens, dev))
        ids_np = w.prefix_blocks()
        nb = int(ids_np.size)
        ids = _i32(ids_np if nb else np.zeros(1, np.int32), dev)
        q = randn(w.T_new, w.Hq, w.d)
        k_new, v_new = randn(w.T_new, w.Hkv, w.d), randn(w.T_new, w.Hkv, w.d)
        img = randn(nb, w.L, 2, w.Hkv, w.ps, w.d) if nb else None
        out = torch.empty_like(q)
        payload = nb * w.page_bytes
        flops = w.attn_flops()

        def step(ev=None):
            if ev:
                ev[0].record(stream)
            if nb:
                gcb.gc_kv_restore(pool.handle, img, ids, nb, stream, None,
                                  gcb.GC_RESTORE_SRC_DEVICE)
            if ev:
                ev[1].record(stream)
            gcb.gc_kv_append(pool.handle, k_new, v_new, bt, pl, stream, 0, cu, w.B, w.max_blocks,
                             w.T_new)
            if ev:
                ev[2].record(stream)
            gcb.gc_prefix_prefill_attn(q, pool.handle, bt, pl, nl, out, stream, 0, cu, w.B,
                                       w.max_blocks, w.Hq, w.scale, w.T_new)
            if ev:
                ev[3].record(stream)

        step_bytes = (2 * q.numel() * 2 + 2 * k_new.numel() * 2 + 2 * payload +
                      int(w.total_lens.sum()) * w.Hkv * w.d * 4)
        flush = step_bytes < 2 * 129 * 2**20
        one = flops / 1e12 / peak_t * 1e3 + 2 * payload / 1e9 / peak_h * 1e3  # ideal ms
        steps = max(3, min(args.config_steps, int(1500 / max(one, 0.01))))
        for _ in range(3):
            step()
        torch.cuda.synchronize()
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(steps)]
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for k in range(steps):
            if flush:
                flush_buf.fill_(k & 0xff)
            step(evs[k])
        b.record(stream)
        torch.cuda.synchronize()
        ms = (statistics.mean(e[0].elapsed_time(e[3]) for e in evs) if flush
              else a.elapsed_time(b) / steps)
        r_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
        ap_ms = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
        at_ms = statistics.mean(e[2].elapsed_time(e[3]) for e in evs)
        # the restore's HBM fraction: back-to-back launches, so each launch's
        # writes left in L2 are written back inside the next one's time (all
        # but the last launch's, at most the 129 MB L2 of >= 10 x 2 x payload)
        rb_ms = None
        if nb:
            reps = max(10, int(math.ceil(10 * 129 * 2**20 / (2 * payload))))
            a.record(stream)
            for _ in range(reps):
                gcb.gc_kv_restore(pool.handle, img, ids, nb, stream, None,
                                  gcb.GC_RESTORE_SRC_DEVICE)
            b.record(stream)
            torch.cuda.synchronize()
            rb_ms = a.elapsed_time(b) / reps
        ok = pool.check(stream) == gcb.GC_OK

        # end to end: pinned host inputs, staged restore, output back, one stream
        q_h, k_h, v_h = (t.cpu().pin_memory() for t in (q, k_new, v_new))
        img_h = img.cpu().pin_memory() if nb else None
        out_h = torch.empty(out.shape, dtype=out.dtype).pin_memory()

        def e2e_step():
            q.copy_(q_h, non_blocking=True)
            k_new.copy_(k_h, non_blocking=True)
            v_new.copy_(v_h, non_blocking=True)
            if nb:
                gcb.gc_kv_restore(pool.handle, img_h, ids, nb, stream, img, 0)
            gcb.gc_kv_append(pool.handle, k_new, v_new, bt, pl, stream, 0, cu, w.B, w.max_blocks,
                             w.T_new)
            gcb.gc_prefix_prefill_attn(q, pool.handle, bt, pl, nl, out, stream, 0, cu, w.B,
                                       w.max_blocks, w.Hq, w.scale, w.T_new)
            out_h.copy_(out, non_blocking=True)

        for _ in range(2):
            e2e_step()
        torch.cuda.synchronize()
        e_steps = max(2, steps // 2)
        a.record(stream)
        for _ in range(e_steps):
            e2e_step()
        b.record(stream)
        torch.cuda.synchronize()
        e2e_ms = a.elapsed_time(b) / e_steps
        ok = ok and pool.check(stream) == gcb.GC_OK
        at_tf = flops / (at_ms / 1e3) / 1e12
        r_gbs = 2 * payload / (r_ms / 1e3) / 1e9 if nb else None
        rb_gbs = 2 * payload / (rb_ms / 1e3) / 1e9 if nb else None
        res[w.name] = {
            "batch": w.B, "new_tokens": w.T_new, "prefix_tokens": int(w.prefix_lens.sum()),
            "page_size": w.ps,
            "attn_kernel": ("attn_tc2_kernel (CTA pairs)" if w.d == 128
                            else f"attn_tc_kernel<{w.d}>"),
            "steps": steps, "ms_per_step": ms, "tok_per_s": w.T_new / (ms / 1e3),
            "attn_ms": at_ms, "attn_tflops": at_tf, "attn_frac_burst": at_tf / peak_t,
            "restore_ms": r_ms if nb else 0.0, "restore_gbs_in_step": r_gbs,
            "restore_gbs": rb_gbs, "restore_frac_hbm": (rb_gbs / peak_h) if nb else None,
            "restore_note": "restore_gbs / restore_frac_hbm: back-to-back launches (L2 write-back "
                            "inside the timing); restore_gbs_in_step: the step's own launch, "
                            "whose writes partly stay in L2",
            "append_ms": ap_ms,
            "e2e_tok_per_s": w.T_new / (e2e_ms / 1e3), "e2e_ms_per_step": e2e_ms,
            "e2e_h2d_bytes_per_step": int((q.numel() + 2 * k_new.numel()) * 2 + payload),
            "e2e_d2h_bytes_per_step": int(out.numel() * 2),
            "e2e_h2d_gbs": ((q.numel() + 2 * k_new.numel()) * 2 + payload) / (e2e_ms / 1e3) / 1e9,
            "e2e_h2d_frac_link": (((q.numel() + 2 * k_new.numel()) * 2 + payload) /
                                  (e2e_ms / 1e3) / 1e9 / link_gbs),
            "link_h2d_gbs": link_gbs,
            "l2": "flushed between steps" if flush else "inputs larger than L2",
            "device_status_ok": ok, "wall_s": time.perf_counter() - t_cfg}
        del q_h, k_h, v_h, img_h, out_h, q, k_new, v_new, img, out
        pool.close()
        torch.cuda.empty_cache()
    return res


def decode_q8_entry(w, db, stream, pk, reps):
    """The same decode step with every full cached page read from an 8-bit
    image (gc_paged_decode_attn_q8); the page holding the new token stays in
    the pool.  Algorithmic bytes: the image pages' codes and scales, the pool
    pages' K and V rows, q and out."""
    import torch

    from paper_2505_23970_gb300 import binding as gcb
    from paper_2505_23970_gb300.harness import _i32

    table = np.full((w.B, w.max_blocks), -1, dtype=np.int32)
    ids = []
    for b in range(w.B):
        full = int(w.prefix_lens[b]) // w.ps
        table[b, :full] = np.arange(len(ids), len(ids) + full)
        ids.extend(w.block_table[b, :full].tolist())
    n = len(ids)
    chunk8 = gcb.gc_kv_q8_chunk_bytes(db.pool.cfg)
    img = torch.empty(max(n, 1) * w.L * 2 * chunk8, dtype=torch.uint8, device=db.q.device)
    gcb.gc_kv_save_q8(db.pool.handle, img, _i32(np.asarray(ids, np.int32), db.q.device), n, 0,
                      w.L, stream, None, gcb.GC_SAVE_DST_DEVICE)
    table_d = _i32(table, db.q.device)
    seq = _i32(w.total_lens, db.q.device)
    need = gcb.gc_paged_decode_workspace_bytes(db.pool.handle, w.B, w.max_blocks, w.Hq)
    wsb = torch.empty(max(need, 16), dtype=torch.uint8, device=db.q.device)
    out = torch.empty_like(db.out)

    def f():
        gcb.gc_paged_decode_attn_q8(db.q, db.pool.handle, db.block_table, seq, out, stream, 0,
                                    w.B, w.max_blocks, w.Hq, w.scale, wsb, need, img, table_d,
                                    n, 0)

    for _ in range(3):
        f()
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(reps):
        f()
    b.record(stream)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / reps
    ok = db.check(stream) == gcb.GC_OK
    img_keys = n * w.ps
    pool_keys = int(w.total_lens.sum()) - img_keys
    byts = (n * 2 * chunk8 + pool_keys * w.Hkv * w.d * 2 * 2 +
            2 * w.B * w.Hq * w.d * 2)
    gbs = byts / (ms / 1e3) / 1e9
    del img, wsb, out
    return {"us_per_step": ms * 1e3, "bytes_per_step": byts, "gbs": gbs,
            "frac_hbm": gbs / pk["hbm_gbs"], "tok_per_s": w.B / (ms / 1e3),
            "image_pages": n, "device_status_ok": ok}


def bench_decode(args, pk):
    """Paged decode attention (one new token per request) on two contexts
    mixes: 8 x 9216 tokens (the 70B prefill config, continued) and the 64
    conversation-mix contexts.  HBM-bound: algorithmic bytes = every context
    key's K and V row once + q + out."""
    import torch

    from paper_2505_23970_gb300 import binding as gcb
    from paper_2505_23970_gb300 import workloads as wl
    from paper_2505_23970_gb300.harness import DeviceBatch

    res = {}
    stream = torch.cuda.current_stream()
    for w in (wl.llama3_70b_decode(seed=args.seed), wl.decode_mix(seed=args.seed)):
        db = DeviceBatch(w)
        db.restore()
        db.append()
        db.decode()
        torch.cuda.synchronize()
        reps = 20
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        for _ in range(3):
            db.decode(stream)
        a.record(stream)
        for _ in range(reps):
            db.decode(stream)
        b.record(stream)
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / reps
        ok = db.check(stream) == gcb.GC_OK
        kv = int(w.total_lens.sum()) * w.Hkv * w.d * 2 * 2
        qo = 2 * w.B * w.Hq * w.d * 2
        gbs = (kv + qo) / (ms / 1e3) / 1e9
        ws = gcb.gc_paged_decode_workspace_bytes(db.pool.handle, w.B, w.max_blocks, w.Hq)
        res[w.name] = {"batch": w.B, "context_tokens": int(w.total_lens.sum()),
                       "us_per_step": ms * 1e3, "bytes_per_step": kv + qo, "gbs": gbs,
                       "frac_hbm": gbs / pk["hbm_gbs"], "tok_per_s": w.B / (ms / 1e3),
                       "workspace_bytes": ws, "device_status_ok": ok}
        res[w.name]["q8"] = decode_q8_entry(w, db, stream, pk, reps)
        db.close()
    return res


def bench_attn_q8(args, pk):
    """Prefill attention over cached pages kept in the 8-bit tier
    (gc_prefix_prefill_attn_q8) on the 70B-shaped layer and the conversation
    mix: every full cached page is read from an INT8 image in device memory
    (made with gc_kv_save_q8) and dequantised in the kernel; partly filled
    last pages, which the new tokens are appended into, stay in the pool.
    Next to it: the pool-only kernel, and the two-step path it replaces
    (gc_kv_restore_q8 of the same pages into the pool, then attention).
    Algorithmic HBM bytes of the cached K/V per step, counting one read
    pass: two-step = image I + pool write B + pool read B; one-step = I, so
    the one-step path moves 2B fewer bytes."""
    import torch

    from paper_2505_23970_gb300 import binding as gcb
    from paper_2505_23970_gb300 import workloads as wl
    from paper_2505_23970_gb300.harness import DeviceBatch, _i32

    res = {}
    stream = torch.cuda.current_stream()
    for w in (wl.llama3_70b_layer(seed=args.seed), wl.conversation_mix(seed=args.seed)):
        db = DeviceBatch(w)
        db.restore()
        db.append()
        table = np.full((w.B, w.max_blocks), -1, dtype=np.int32)
        ids = []
        for b in range(w.B):
            full = int(w.prefix_lens[b]) // w.ps
            table[b, :full] = np.arange(len(ids), len(ids) + full)
            ids.extend(w.block_table[b, :full].tolist())
        n = len(ids)
        ids_d = _i32(np.asarray(ids, dtype=np.int32), db.q.device)
        table_d = _i32(table, db.q.device)
        chunk8 = gcb.gc_kv_q8_chunk_bytes(db.pool.cfg)
        img = torch.empty(max(n, 1) * w.L * 2 * chunk8, dtype=torch.uint8, device=db.q.device)
        gcb.gc_kv_save_q8(db.pool.handle, img, ids_d, n, 0, w.L, stream, None,
                          gcb.GC_SAVE_DST_DEVICE)
        out_q8 = torch.empty_like(db.out)

        def attn_q8():
            gcb.gc_prefix_prefill_attn_q8(db.q, db.pool.handle, db.block_table, db.prefix_lens,
                                          db.new_lens, out_q8, stream, 0, db.cu_new_lens, w.B,
                                          w.max_blocks, w.Hq, w.scale, w.T_new, img, table_d,
                                          n, 0)

        def two_step():
            gcb.gc_kv_restore_q8(db.pool.handle, img, ids_d, n, 0, w.L, stream, None,
                                 gcb.GC_RESTORE_SRC_DEVICE)
            db.attn(stream)

        def timed(fn, reps=10):
            for _ in range(3):
                fn()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(reps):
                fn()
            b.record(stream)
            torch.cuda.synchronize()
            return a.elapsed_time(b) / reps

        ms_pool = timed(lambda: db.attn(stream))
        ms_q8 = timed(attn_q8)
        ms_two = timed(two_step)
        same = bool(torch.equal(out_q8.view(torch.int16), db.out.view(torch.int16)))
        ok = db.check(stream) == gcb.GC_OK
        flops = w.attn_flops()
        B_bytes = n * w.L * 2 * w.Hkv * w.ps * w.d * 2
        I_bytes = n * w.L * 2 * chunk8
        tf = flops / (ms_q8 / 1e3) / 1e12
        res[w.name] = {
            "image_pages": n, "image_bytes": I_bytes, "cached_kv_bf16_bytes": B_bytes,
            "hbm_bytes_saved_per_step": 2 * B_bytes,
            "ms": {"attn_q8": ms_q8, "attn_pool": ms_pool, "restore_q8_then_attn": ms_two},
            "attn_q8_tflops": tf, "attn_q8_frac_of_measured_peak": tf / pk["bf16_tflops"],
            "attn_pool_tflops": flops / (ms_pool / 1e3) / 1e12,
            "speedup_vs_two_step": ms_two / ms_q8,
            "bit_identical_to_two_step": same, "device_status_ok": ok,
            "l2": "not flushed between launches (image and pool pages exceed L2 on the 70B "
                  "layer; the mix's 64 requests fit partly)"}
        del img, out_q8
        db.close()
        torch.cuda.empty_cache()
    return res


def bench_ttft80(args, image=None):
    """All 80 layers of one request with an 8192-token cached prefix and
    1024 new tokens: restore of each layer's cached pages (pinned host ->
    staging -> pool) + append + attention, with the restores pipelined on a
    side stream (event per layer) against the layers' compute, next to the
    same work done one after the other, each half alone, and a from-scratch
    prefill of the whole 9216-token context (append + attention over all
    layers, no restore).  The attention-and-restore analogue of time to
    first token with and without the cache (no projections or MLPs)."""
    import torch

    from paper_2505_23970_gb300 import binding as gcb
    from paper_2505_23970_gb300 import workloads as wl
    from paper_2505_23970_gb300.harness import LayerStack

    w = wl.llama3_70b_80layer_prefill(seed=args.seed)
    if image is not None and image.shape[:2] == (int(w.prefix_blocks().size), w.L):
        w._cache["src"] = image  # same shape: reuse the 80-layer image already made
    wr = wl.llama3_70b_80layer_prefill(seed=args.seed, recompute=True)
    cached, scratch = LayerStack(w), LayerStack(wr)
    stream = torch.cuda.current_stream()
    reps = 5

    def timed(fn):
        """Median over `reps` runs, each bracketed by its own events (the
        host link is shared with other jobs on the machine, and one slow
        run should not move the figure)."""
        for _ in range(2):
            fn()
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(reps)]
        for a, b in evs:
            a.record(stream)
            fn()
            b.record(stream)
        torch.cuda.synchronize()
        return statistics.median(a.elapsed_time(b) for a, b in evs)

    def restore_layers():
        for l in range(w.L):
            cached.restore_layer(l, stream)

    def stage_layers():
        for l in range(w.L):
            cached.stage_layer(l, stream)

    def traced():
        """One copy-stream pipelined run with per-layer events: when each
        layer's copy landed, when its scatter and its attention finished."""
        tr = {}
        t0 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        cached.run(pipelined=True, trace=tr)
        torch.cuda.synchronize()
        at = {k: [t0.elapsed_time(e) for e in v] for k, v in tr.items()}
        # main-stream time spent waiting for a copy: scatter l started when
        # both layer l-1's attention and layer l's copy were done
        waits = [max(0.0, at["copied"][l] - (at["computed"][l - 1] if l else 0.0))
                 for l in range(w.L)]
        return {"copies_done_ms": at["copied"][-1], "compute_done_ms": at["computed"][-1],
                "main_waited_for_copies_ms": sum(waits),
                "layers_waiting_for_their_copy": sum(1 for x in waits if x > 0.005),
                "copied_ms_first_8": at["copied"][:8], "computed_ms_first_8": at["computed"][:8],
                "scatter_ms_mean": statistics.mean(
                    at["scattered"][l] - max(at["copied"][l], at["computed"][l - 1] if l else 0.0)
                    for l in range(w.L))}

    ms = {}
    cached.restore_all(stream)
    cached.use_q8()      # 8-bit cache tier: the same pages as an INT8 image
    ms["pipelined_q8"] = timed(lambda: cached.run(pipelined=True))
    ms["pipelined_q8_graph"] = timed(cached.capture(pipelined=True).replay)
    ms["restore_per_layer_only_q8"] = timed(restore_layers)
    ms["stage_only_q8"] = timed(stage_layers)
    cached.q8 = False
    # the whole copy-stream pipeline recorded once into a CUDA graph
    ms["pipelined_graph"] = timed(cached.capture(pipelined=True).replay)
    ms.update({
        "pipelined": timed(lambda: cached.run(pipelined=True)),
        "pipelined_side_restore": timed(lambda: cached.run(pipelined=True,
                                                           schedule="side-restore")),
        "sequential": timed(lambda: cached.run(pipelined=False)),
        "restore_per_layer_only": timed(restore_layers),
        "stage_only": timed(stage_layers),
        "restore_whole_only": timed(lambda: cached.restore_all(stream)),
        "prefill_only": timed(cached.prefill_only),
        "recompute": timed(scratch.prefill_only),
    })
    # the host link's rate varies between runs (other work on the host):
    # keep the fastest of three traced runs
    trace = min((traced() for _ in range(3)), key=lambda t: t["compute_done_ms"])
    ok = cached.check() == gcb.GC_OK and scratch.check() == gcb.GC_OK
    cached.close()
    scratch.close()
    # the restore work the pipeline has to hide: every layer's copy (the
    # link) plus its scatter; hidden = what the pipelined run saves over
    # doing that and the compute one after the other
    restore_ms = ms["restore_whole_only"]
    hidden = restore_ms + ms["prefill_only"] - ms["pipelined"]
    return {
        "workload": "llama3-70b-80layer: 1 request, cached prefix 8192, 1024 new tokens, "
                    "64 q / 8 kv heads, d 128, ps 16; restore from pinned host",
        "schedule": "pipelined: every layer's host->device copy on a copy stream up front, "
                    "layer l's scatter + append + attention on the compute stream after "
                    "layer l's copy event; pipelined_side_restore: one staged "
                    "restore_layers call per layer on a side stream; *_graph: the copy-stream "
                    "schedule recorded into a CUDA graph and replayed; each figure the "
                    "median of 5 runs, each run timed by its own events",
        "device_status_ok": ok, "ms": ms, "trace": trace,
        "restore_hidden_frac": hidden / restore_ms,
        "pipelined_over_bound": ms["pipelined"] / max(ms["stage_only"], ms["prefill_only"]),
        "speedup_vs_recompute": ms["recompute"] / ms["pipelined"],
        "speedup_vs_recompute_q8": ms["recompute"] / ms["pipelined_q8"],
        "restore_bytes": int(w.prefix_blocks().size) * w.page_bytes,
        "gpu_launches_pipelined": 3 * w.L,
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="70b",
                    help="70b (default), 8b, tiny, mix<p>, long, long-recompute")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-restore80", action="store_true")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-q8-attn", action="store_true",
                    help="skip attention over 8-bit pages")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the per-configuration measurements of every workload")
    ap.add_argument("--config-steps", type=int, default=10,
                    help="timed steps per configuration in the per-configuration section")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--ref-step-seconds", type=float, default=None,
                    help="oracle seconds per step of --impl reference (default: sized so "
                         "the whole run takes about 2.5 minutes)")
    ap.add_argument("--only", choices=["decode", "restore80", "prefill80", "configs", "q8attn"],
                    default=None,
                    help="run one secondary measurement alone and print it (for profilers)")
    ap.add_argument("--profile", action="store_true",
                    help="timed loop only (for ncu launch lists): no e2e, clocks or baselines")
    args = ap.parse_args()
    if args.warmup < 3 and not args.profile:
        ap.error("--warmup must be >= 3")
    global WORKLOAD
    WORKLOAD = {"70b": "llama3-70b-layer", "8b": "llama3-8b-layer", "tiny": "tiny",
                "long": "long-document", "long-recompute": "long-document-recompute"}.get(
                    args.config, f"conversation-{args.config}")
    if args.only:
        import torch
        torch.cuda.set_device(0)
        pk = peaks()
        if args.only == "decode":
            print(json.dumps({"decode": bench_decode(args, pk)}), flush=True)
        elif args.only == "q8attn":
            print(json.dumps({"attn_q8": bench_attn_q8(args, pk)}), flush=True)
        elif args.only == "configs":
            print(json.dumps({"configs": bench_configs(args, pk)}), flush=True)
        elif args.only == "restore80":
            print(json.dumps({"restore_80layer": bench_restore80(args, pk)[1]}), flush=True)
        else:
            print(json.dumps({"prefill_80layer": bench_ttft80(args)}), flush=True)
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
