#!/usr/bin/env python3
"""Throughput of the LaCache two-stage lookahead lookup on GB300.

    python bench.py [--gpus N --steps K --warmup W] [--workload large-16m] [--stage1 auto|tensor|stream]
    python bench.py --impl reference ...        # the fp64 oracle on the host cores, a bounded sample per step

A step is one lookup: stage 1 (key check with fused threshold + top-c) and stage 2 (merge, lookahead check,
decision) for one batch of B synthetic queries against a resident cache of N entries. The default workload is the
largest single-GPU one: 16,777,216 entries of d = 1024 (34.4 GB of keys, 69.8 GB of store) and batches of 128
queries. The inputs are resident in HBM before timing starts. Every step reads the whole key store, far larger
than L2, so no L2 flush is needed between steps. Where a step streams less than twice the L2 (the SimHash index of a
1M-entry store, a 4k-entry store), a write of four times the L2 runs between timed steps, every step is timed on its
own and the end-to-end calls are timed one by one after a flush (`L2Flush`). The device time is taken with CUDA
events on the launching stream, between barriers, as the max over ranks.

With N > 1 GPUs, one process runs per GPU. Under torchrun (WORLD_SIZE set) this script is one of the ranks;
otherwise `--gpus N` builds the library once and starts N ranks through torch.distributed.run itself. Every rank
serves its own replica of the cache with its own query stream: the units are independent lookups, with no
collective on the data path (weak scaling). `--mode shard` splits the store by entry range instead.

Rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "lookups/sec at 1 GB300 (N entries, batch B, k) + % of HBM or bf16 roofline"
UNIT = "queries/s"
FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
STAGE1_SOURCES = {"tensor": "stage1_tensor.cu", "tensor-pair": "stage1_tensor.cu", "stream": "stage1_stream.cu",
                  "lsh": "lsh.cu", "lsh-tensor": "lsh_tc.cu"}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="large-16m")
    ap.add_argument("--stage1", choices=["auto", "tensor", "stream", "lsh"], default="auto")
    ap.add_argument("--lsh-bits", type=int, default=256, help="SimHash signature bits for --stage1 lsh")
    ap.add_argument("--batches", type=int, default=8, help="distinct query batches cycled through")
    ap.add_argument("--e2e-steps", type=int, default=500)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--mode", choices=["replicas", "shard"], default="replicas",
                    help="replicas: every rank serves its own batches against a full copy of the store (weak "
                         "scaling); shard: the store is split by entry range across the ranks, every rank serves "
                         "the same batches, one all-gather and a merge per lookup (strong scaling)")
    ap.add_argument("--entries", type=int, default=0,
                    help="store size override: a smaller case of the workload (profiling captures)")
    ap.add_argument("--batch", type=int, default=0,
                    help="batch size override: a batch-size case of the workload (kernel crossover measurements)")
    return ap.parse_args()


def rank_info():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


def launch_ranks(n: int, argv: list[str]) -> int:
    """Run this script on n ranks of this node, one process per GPU, through torch.distributed.run. The ranks
    inherit stdout, so rank 0's JSON line is this process's output."""
    import socket
    with socket.socket() as sock:
        sock.bind(("127.0.0.1", 0))
        port = sock.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={n}",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.abspath(__file__), *argv]
    return subprocess.call(cmd)


def peaks_lib():
    """The measurement kernels (libpeaks.so, built beside the lookup library)."""
    from paper_2608_01718_gb300 import build
    lib = ctypes.CDLL(build.PEAKS_LIB)
    lib.lcpeaks_read.argtypes = [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p]
    lib.lcpeaks_popc.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_void_p, ctypes.c_int,
                                 ctypes.c_void_p]
    return lib


class L2Flush:
    """Keeps a step's inputs out of L2 between timed steps when they would fit in it. A step that streams fewer
    than twice the L2's bytes (streamed_bytes) gets a write of four times the L2 before it: a fill of a device
    buffer, on the current stream, outside the step's own events. Otherwise the flush does nothing."""

    def __init__(self, streamed_bytes: int, what: str):
        import torch
        props = torch.cuda.get_device_properties(torch.cuda.current_device())
        self.l2 = int(getattr(props, "L2_cache_size", 0) or 129 * 10**6)
        self.on = streamed_bytes < 2 * self.l2
        self.buf = torch.empty(4 * self.l2, dtype=torch.uint8, device="cuda") if self.on else None
        self.fills = 0
        self.note = (f"flush: the {what} read per step ({streamed_bytes / 1e6:.1f} MB) fit in the "
                     f"{self.l2 / 1e6:.0f} MB L2, so a {4 * self.l2 / 1e6:.0f} MB write runs before every timed step "
                     "(outside its events) and before every timed end-to-end call (outside its clock)"
                     if self.on else
                     f"no flush: the {what} read per step ({streamed_bytes / 1e9:.2f} GB) exceed twice the "
                     f"{self.l2 / 1e6:.0f} MB L2")

    def __call__(self):
        if self.on:
            self.fills += 1
            self.buf.fill_(self.fills & 0xFF)


def device_steps_ms(step, steps: int, stream, flush: L2Flush) -> float:
    """Device time (ms) of steps 0 .. steps-1 on `stream`: one event pair around the whole loop, or, with the L2
    flush on, one pair around each step with the flush between them, summed."""
    import torch
    if not flush.on:
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record(stream)
        for i in range(steps):
            step(i)
        ev1.record(stream)
        torch.cuda.synchronize()
        return ev0.elapsed_time(ev1)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for i in range(steps):
        flush()
        evs[i][0].record(stream)
        step(i)
        evs[i][1].record(stream)
    torch.cuda.synchronize()
    return sum(a.elapsed_time(b) for a, b in evs)


def timed_best(launch, reps: int = 5) -> float:
    """Best CUDA-event time (ms) of `launch` on the current stream, over reps runs after one warm-up run."""
    import torch
    best = float("inf")
    for i in range(reps + 1):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        launch()
        e1.record()
        torch.cuda.synchronize()
        if i:
            best = min(best, e0.elapsed_time(e1))
    return best


def read_peak_gbs() -> float:
    """HBM read rate of a kernel that only reads: the best of 5 CUDA-event-timed passes of lcpeaks_read (128-bit
    loads, four in flight per thread) over a 4 GiB buffer."""
    import torch
    lib = peaks_lib()
    nbytes = 1 << 32
    buf = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    sink = torch.zeros(1, dtype=torch.int32, device="cuda")
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    stream = torch.cuda.current_stream().cuda_stream

    def launch():
        if lib.lcpeaks_read(buf.data_ptr(), nbytes, sink.data_ptr(), sms, stream):
            raise RuntimeError("lcpeaks_read failed")
    ms = timed_best(launch)
    del buf
    torch.cuda.empty_cache()
    return nbytes / (ms / 1e3) / 1e9


def popc_peak(words: int, radius: int) -> dict:
    """The SimHash scan's distance arithmetic with no memory traffic (lcpeaks_popc), timed with CUDA events while
    nvidia-smi samples the SM clock: signature words compared per second, and per clock and SM."""
    import torch
    lib = peaks_lib()
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    sink = torch.zeros(1, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    steps = 4096 * 8 // words
    clocks = ClockSampler(torch.cuda.current_device())
    clocks.start()

    def launch():
        if lib.lcpeaks_popc(words, steps, radius, sink.data_ptr(), sms, stream):
            raise RuntimeError("lcpeaks_popc failed")
    ms = timed_best(launch, reps=10)
    clk = clocks.stop()
    total = 2 * sms * 512 * steps * 32 * words
    rate = total / (ms / 1e3)
    mhz = clk.get("sm_mhz") or 2070.0
    return {"words_per_s": rate, "words_per_clock_per_sm": rate / (sms * mhz * 1e6), "sm_mhz": mhz}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return json.load(f), "measured"
    return dict(FALLBACK), "fallback"


class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons while the timed region runs."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        self.proc.wait()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9 and parts[1].replace(".", "").isdigit():
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(float(r[1]) for r in rows),
                "sm_max_mhz": max(float(r[2]) for r in rows),
                "power_w_max": max(float(r[3]) for r in rows if r[3].replace(".", "").isdigit()) if rows else None,
                "reasons": reasons, "samples": len(rows)}


def algorithmic(w, batch):
    """Bytes and flops the method must move / do per lookup (keys read once, c candidate rows gathered)."""
    stage1_bytes = w.n * w.d * 2 + batch * w.d * 2
    stage2_bytes = batch * w.top_c * (2 * w.pd + 4 * w.k) + batch * (2 * w.pd + 4 * w.k)
    flops = 2 * batch * w.n * w.d + 2 * batch * w.top_c * w.pd
    return stage1_bytes, stage2_bytes, flops


def kernel_traffic(stage1: str, workload: str, variant: str = ""):
    """DRAM bytes per launch of the stage-1 kernel from the committed ncu capture, if the kernel source has not
    changed since the capture (else None). `variant` names a setting the traffic depends on (the SimHash
    signature width)."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        rec = json.load(f).get(f"stage1_{stage1}{variant}/{workload}")
    if not rec:
        return None
    src = os.path.join(ROOT, "paper_2608_01718_gb300", "csrc", STAGE1_SOURCES[stage1])
    with open(src, "rb") as f:
        if hashlib.sha256(f.read()).hexdigest() != rec.get("source_sha256"):
            return None
    return rec.get("dram_bytes_per_launch")


def cpu_threads() -> int:
    for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(var, "").isdigit():
            return int(os.environ[var])
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def oracle_sample(w, rows: int, offset: int = 0, device="cpu"):
    """Host bytes of store rows [offset, offset + rows) (regenerated chunk by chunk) and of query batch 0."""
    import numpy as np

    import oracle
    from paper_2608_01718_gb300 import workloads as wl
    keys, pres, ids = [], [], []
    got = 0
    index = offset // wl.CHUNK_ROWS
    start = offset - index * wl.CHUNK_ROWS
    while got < rows:
        ch = wl.store_chunk(w, index, device)
        take = min(rows - got, ch["key"].shape[0] - start)
        sl = slice(start, start + take)
        if w.key_dtype == "f32":
            keys.append(oracle.round_to_bf16(wl.f32_array(ch["key"][sl])))
            pres.append(oracle.round_to_bf16(wl.f32_array(ch["prefix"][sl])))
        else:
            keys.append(wl.bf16_bits(ch["key"][sl]))
            pres.append(wl.bf16_bits(ch["prefix"][sl]))
        ids.append(ch["ids"][sl].cpu().numpy())
        got += take
        index += 1
        start = 0
    store = oracle.Store.of(np.concatenate(keys), np.concatenate(pres), np.concatenate(ids))
    q = wl.batch(w, 0, device)
    oq = {"emb": wl.bf16_bits(q["emb"]), "prefix": wl.bf16_bits(q["prefix"]), "ids": q["ids"].cpu().numpy()}
    return store, oq


def time_oracle(store, oq, w) -> float:
    """Seconds the oracle takes to look up the whole batch against the given store rows."""
    import oracle
    p = oracle.Params(w.tau_c, w.tau_a, w.top_c, prefix_dims=w.prefix_dims, tau_a_models=w.tau_a_models)
    t0 = time.perf_counter()
    oracle.lookup(store, oq, p)
    return time.perf_counter() - t0


def gen_device():
    import torch
    return "cuda" if torch.cuda.is_available() else "cpu"


def run_reference(args, w):
    rank, _, world = rank_info()
    if rank != 0:
        return 0
    dev = gen_device()
    # size the per-step sample so that warm-up + timed steps take about two minutes in all
    probe_rows = min(w.n, 16384)
    store, oq = oracle_sample(w, probe_rows, 0, dev)
    per_row = time_oracle(store, oq, w) / probe_rows
    budget = 120.0 / max(1, args.steps + args.warmup)
    rows = int(min(w.n, max(2048, budget / per_row)))
    store, oq = oracle_sample(w, rows, 0, dev)
    total = 0.0
    for i in range(args.warmup + args.steps):
        t = time_oracle(store, oq, w)
        if i >= args.warmup:
            total += t
    sec_per_batch_full = total / args.steps * (w.n / rows)
    value = w.batch / sec_per_batch_full
    cores = cpu_threads()
    sample = (f"each step: oracle lookup of the {w.batch}-query batch against the first {rows} of the {w.n} "
              f"store rows; value scaled to the full store by N/rows (the oracle's work is linear in N)")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(w) | {"parallelism": "single",
                                            "l2": "not applicable: the oracle runs on the host cores"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def combine_ranks(elapsed_ms: float, e2e_s: float, world: int, steps: int, e2e_steps: int, batch: int,
                  device=None) -> dict:
    """Whole-job numbers from every rank's own timings: the slowest rank's time (all ranks started together after
    a barrier) and the queries all ranks processed. With one rank no process group is needed."""
    if world > 1:
        import torch
        import torch.distributed as dist
        t = torch.tensor([elapsed_ms, e2e_s], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        elapsed_ms, e2e_s = float(t[0]), float(t[1])
    return {"elapsed_ms": elapsed_ms, "e2e_s": e2e_s,
            "value": world * steps * batch / (elapsed_ms / 1e3),
            "e2e_value": world * e2e_steps * batch / e2e_s}


def workload_config(w):
    cfg = {"workload": w.name, "entries": w.n, "d": w.d, "k": w.k, "batch": w.batch, "top_c": w.top_c,
           "tau_c": w.tau_c, "tau_a": w.tau_a, "store_bytes": w.store_bytes}
    if w.prefix_dims is None:
        cfg["mix_near_random_collision"] = list(w.mix)
    else:
        cfg |= {"prefix_dims": list(w.prefix_dims), "tau_a_models": list(w.tau_a_models),
                "mix_near_random_collision_mimic": list(w.mix)}
    return cfg


def run_ours(args, w):
    import torch
    import torch.distributed as dist

    from paper_2608_01718_gb300 import build
    from paper_2608_01718_gb300 import lacache as L
    from paper_2608_01718_gb300 import workloads as wl

    rank, local_rank, world = rank_info()
    torch.cuda.set_device(local_rank)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    build.build()
    stage1 = {"auto": L.LACACHE_STAGE1_AUTO, "tensor": L.LACACHE_STAGE1_TENSOR, "stream": L.LACACHE_STAGE1_STREAM,
              "lsh": L.LACACHE_STAGE1_LSH}
    # A workload with a step count is a serve loop (Algorithm 1 batch by batch): every timed step looks up a fresh
    # batch and then appends its misses, so the store grows while it is timed; the capacity holds that growth.
    serve = w.steps > 1
    warm = max(3, args.warmup)
    capacity = w.n + (warm + args.steps) * w.batch if serve else w.n
    cache = L.LaCache(w.d, w.k, capacity, w.tau_c, w.tau_a, w.top_c, max_batch=w.batch, device=local_rank,
                      stage1=stage1[args.stage1], prefix_dims=w.prefix_dims, tau_a_models=w.tau_a_models)
    dtype = L.LACACHE_F32 if w.key_dtype == "f32" else L.LACACHE_BF16
    for ch in wl.iter_store(w, "cuda"):
        cache.insert(ch["key"], ch["prefix"], ch["ids"], dtype)
        del ch
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    lsh = None
    if args.stage1 == "lsh":
        lsh = {"bits": args.lsh_bits, "radius": wl.lsh_radius(w.tau_c, args.lsh_bits)}
        L.lacache_enable_lsh(cache.h, lsh["bits"], lsh["radius"], wl.hyperplanes(lsh["bits"], w.d, device="cuda"))
        torch.cuda.synchronize()
    nb = args.batches
    batches = [wl.batch(w, step=(rank * nb + i), device="cuda") for i in range(nb)]
    outs = [L.alloc_result(w.batch, w.top_c, "cuda", candidates=False) for _ in range(nb)]
    stream = torch.cuda.current_stream()

    def step(i):
        q = batches[i % nb]
        L.lacache_lookup(cache.h, q["emb"], q["prefix"], q["ids"], outs[i % nb], stream)

    if serve:
        # distinct batches for the warm-up and timed steps, generated before timing starts
        serve_batches = [wl.batch(w, step=i, device="cuda") for i in range(warm + args.steps)]

        def serve_step(i):
            q = serve_batches[i]
            out = outs[i % nb]
            L.lacache_lookup(cache.h, q["emb"], q["prefix"], q["ids"], out, stream)
            cache.append_misses(q["emb"], q["prefix"], q["ids"], out["status"], stream)   # synchronizes

    for i in range(warm):
        (serve_step if serve else step)(i)
    torch.cuda.synchronize()
    cache.sync()
    n_timed_begin = cache.size
    kernel_name = {L.LACACHE_STAGE1_TENSOR: "tensor", L.LACACHE_STAGE1_TENSOR_PAIR: "tensor-pair",
                   L.LACACHE_STAGE1_STREAM: "stream", L.LACACHE_STAGE1_LSH: "lsh",
                   L.LACACHE_STAGE1_LSH_TENSOR: "lsh-tensor"}[cache.last_launch()[1]]
    # what a step streams: the SimHash index (bits / 8 bytes an entry for the popcount scan, bits bytes for the
    # tensor-core scan's expanded copy) or the keys
    if lsh:
        flush = L2Flush(w.n * lsh["bits"] // (1 if kernel_name == "lsh-tensor" else 8), "SimHash index bytes")
    else:
        flush = L2Flush(w.n * w.d * 2, "keys")
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(torch.cuda.current_device())
    clocks.start()
    elapsed_ms = device_steps_ms(lambda i: serve_step(warm + i) if serve else step(i), args.steps, stream, flush)
    if world > 1:
        dist.barrier()
    clock = clocks.stop()
    cache.sync()
    n_timed_end = cache.size
    # Second pass over the same steps with the library's stage events (recorded on the lookup's stream around
    # each kernel) for the per-kernel times of the roofline. The events sit between the two kernels, so this pass
    # is kept out of the throughput measurement above.
    L.lacache_stage_timing(cache.h, args.steps)
    for i in range(args.steps):
        flush()
        step(i)
    t1_ms, t2_ms, timed = L.lacache_stage_times(cache.h)
    L.lacache_stage_timing(cache.h, 0)

    # End to end through the C ABI's host-buffer entry points: every step's batch goes from pinned host memory to
    # the device, the lookup runs, and its decisions come back to pinned host memory, where the host reads them.
    # The arguments of each call are built once, so the loops measure the library calls rather than Python
    # argument marshalling. Two forms are timed:
    #   e2e       lacache_lookup_host_async with two lookups in flight (the serving pattern): the host reads step
    #             i's decisions after an event recorded behind it, while step i + 1 runs;
    #   e2e_sync  lacache_lookup_host, one synchronous call per step.
    depth = 2
    hq = [{k: batches[i][k].cpu().pin_memory() for k in ("emb", "prefix", "ids")} for i in range(nb)]
    hout = [L.alloc_result(w.batch, w.top_c, "cpu", candidates=False, pinned=True) for _ in range(depth)]
    status_np = [o["status"].numpy() for o in hout]
    lib = L.load()
    results = [L._result_struct(o) for o in hout]
    calls = [[(cache.h, w.batch, hq[i]["emb"].data_ptr(), hq[i]["prefix"].data_ptr(), hq[i]["ids"].data_ptr(),
               ctypes.byref(results[slot]), stream.cuda_stream) for slot in range(depth)] for i in range(nb)]
    events = [torch.cuda.Event() for _ in range(depth)]

    def run_async(n: int) -> int:
        bad, served = 0, 0
        for i in range(n):
            slot = i % depth
            if i >= depth:
                events[slot].synchronize()
                served += int(status_np[slot].sum())    # the host reads step i - depth's decisions
            bad |= lib.lacache_lookup_host_async(*calls[i % nb][slot])
            events[slot].record(stream)
        for i in range(max(0, n - depth), n):
            events[i % depth].synchronize()
            served += int(status_np[i % depth].sum())
        if bad:
            raise RuntimeError("lacache_lookup_host_async failed")
        return served

    def run_sync(n: int) -> float:
        """Seconds of n synchronous calls; with the L2 flush on, each call is timed alone after a flush that has
        finished, and the calls' times are summed."""
        bad, total = 0, 0.0
        t0 = time.perf_counter()
        for i in range(n):
            if flush.on:
                flush()
                torch.cuda.synchronize()
                t0 = time.perf_counter()
            bad |= lib.lacache_lookup_host(*calls[i % nb][i % depth])
            if flush.on:
                total += time.perf_counter() - t0
        if bad:
            raise RuntimeError("lacache_lookup_host failed")
        return total if flush.on else time.perf_counter() - t0

    run_sync(max(3, args.warmup))
    if world > 1:
        dist.barrier()
    e2e_sync_s = run_sync(args.e2e_steps)
    sync_status = [o["status"].clone() for o in hout]
    run_async(max(3, args.warmup))
    if world > 1:
        dist.barrier()
    t0 = time.perf_counter()
    run_async(args.e2e_steps)
    e2e_s = time.perf_counter() - t0
    if flush.on:
        # the pipelined loop overlaps calls, so a flush between them cannot be kept out of its clock: the
        # end-to-end figure is then the synchronous calls', each from a flushed L2 (the loop above still checks
        # that pipelined lookups decide as the synchronous ones)
        e2e_s = e2e_sync_s
    # both timed loops ran the same e2e_steps steps, so each output slot's last batch is the same in both: the
    # pipelined lookups must have written the same decisions as the synchronous ones
    for slot in range(depth):
        if not torch.equal(hout[slot]["status"], sync_status[slot]):
            raise RuntimeError("the pipelined host lookups disagree with the synchronous ones")
    sync_job = combine_ranks(elapsed_ms, e2e_sync_s, world, args.steps, args.e2e_steps, w.batch, device="cuda")
    job = combine_ranks(elapsed_ms, e2e_s, world, args.steps, args.e2e_steps, w.batch, device="cuda")
    elapsed_ms, e2e_s = job["elapsed_ms"], job["e2e_s"]
    h2d = w.batch * (2 * w.d + 2 * w.pd + w.k * 4)
    d2h = w.batch * (4 + 1 + 4 + 4 + 4 + 4)

    peaks, peak_src = load_peaks()
    # a serve loop scans a growing store: the stage-timing pass ran on the store as the timed steps left it
    w_alg = w.scaled(n=n_timed_end) if serve else w
    s1_bytes, s2_bytes, flops = algorithmic(w_alg, w.batch)
    t1_avg_s = t1_ms / max(1, timed) / 1e3
    traffic = None if args.entries or args.batch else kernel_traffic(kernel_name, w.name,
                                                                      f"-b{lsh['bits']}" if lsh else "")
    value = job["value"]
    # the stage-1 kernel is bound by HBM below the ridge (flops per byte of the measured peaks), else by the
    # tensor pipe; a kernel timed back to back for over a second is compared with the sustained bf16 peak
    ridge = peaks["bf16_tflops"] * 1e12 / (peaks["hbm_gbs"] * 1e9)
    if lsh and kernel_name == "lsh-tensor":
        # The tensor-core SimHash scan streams the expanded index, N x bits bytes per lookup (one byte per signature
        # bit), and is bound by HBM; the admitted key rows it gathers are not counted.
        index_bytes = w.n * lsh["bits"]
        roof = {"bound": "hbm", "achieved": index_bytes / t1_avg_s / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "peak_source": f"{peak_src} (copy bandwidth)", "algorithmic_index_bytes_per_launch": index_bytes}
    elif lsh:
        # The SimHash scan is bound by integer work on its B x N x (bits / 32) signature-word comparisons per
        # lookup. Population count runs at 16 per clock per SM (the CUDA arithmetic-throughput table), the logic
        # and integer operations at 64. The scan's carry-save adders fold 8 words into 5 popcounts (4 into 3), whose
        # 19 (10) other operations fit under the popcount time on the 64-wide pipe. So the derived ceiling is
        # 16 x 8 / 5 words (16 x 4 / 3 at 128 bits) per clock per SM x SMs x the maximum SM clock. Beside it, the
        # same arithmetic measured with no memory traffic (lcpeaks_popc), scaled to the scan's median SM clock.
        # With few queries the scan is bound by streaming the index (N x bits / 8 bytes) instead: the roofline
        # takes whichever of the two times is longer at the peaks, and the line keeps both rates.
        sms = torch.cuda.get_device_properties(local_rank).multi_processor_count
        words = w.batch * w.n * (lsh["bits"] // 32)
        per_clock = 16 * (8 / 5 if (lsh["bits"] // 32) % 8 == 0 else 4 / 3)
        achieved = words / t1_avg_s / 1e12
        mp = popc_peak(lsh["bits"] // 32, lsh["radius"])
        measured = mp["words_per_clock_per_sm"] * sms * (clock.get("sm_mhz") or mp["sm_mhz"]) * 1e6 / 1e12
        alu_peak = per_clock * sms * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12
        index_bytes = w.n * lsh["bits"] // 8
        alu = {"achieved": achieved, "peak": alu_peak, "unit": "Twords/s",
               "algorithmic_index_bytes_per_launch": index_bytes,
               "peak_source": f"derived: {per_clock:.1f} signature words/clock/SM (popcounts at 16/clock after "
                              f"carry-save folding) x {sms} SMs x max SM clock",
               "measured_peak": measured, "frac_of_measured_peak": achieved / measured,
               "measured_peak_source": "lcpeaks_popc: the scan's XOR / carry-save / popcount / compare arithmetic "
                                       f"on register and shared data, {mp['words_per_clock_per_sm']:.2f} words/clock"
                                       "/SM measured, x SMs x the scan's median SM clock",
               "algorithmic_word_comparisons_per_launch": words,
               "note": "the work counts every signature word of every (query, entry) pair, as a brute-force "
                       "comparison would; the scan's prefix test reads only the first 3/4, 5/8 or 1/2 of the "
                       "words of the pairs it rejects there (exactly: a prefix distance above the radius settles "
                       "the pair), so the achieved rate can reach or pass the arithmetic peak"}
        if index_bytes / (peaks["hbm_gbs"] * 1e9) > words / (alu_peak * 1e12):
            roof = {"bound": "hbm", "achieved": index_bytes / t1_avg_s / 1e9, "peak": peaks["hbm_gbs"],
                    "unit": "GB/s", "peak_source": f"{peak_src} (copy bandwidth)",
                    "algorithmic_index_bytes_per_launch": index_bytes,
                    "algorithmic_word_comparisons_per_launch": words,
                    "time_covers": "the query-signature kernel and the scan (stage 1)",
                    "alu": alu | {"frac": achieved / alu_peak}}
        else:
            roof = {"bound": "alu", **alu}
    elif flops / s1_bytes < ridge:
        roof = {"bound": "hbm", "achieved": s1_bytes / t1_avg_s / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "peak_source": f"{peak_src} (copy bandwidth)"}
    else:
        sustained = elapsed_ms > 1000.0 and "bf16_tflops_sustained" in peaks
        peak = peaks["bf16_tflops_sustained"] if sustained else peaks["bf16_tflops"]
        roof = {"bound": "tensor", "achieved": flops / t1_avg_s / 1e12, "peak": peak, "unit": "TFLOP/s",
                "peak_source": f"{peak_src} ({'sustained' if sustained else 'burst'} bf16 dense)"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    if roof["bound"] == "hbm":
        # beside the copy peak (which reads and writes every byte), the rate of a kernel that only reads
        rp = read_peak_gbs()
        roof |= {"read_peak_gbs": rp, "frac_of_read_peak": roof["achieved"] / rp,
                 "read_peak_source": "measured live: lcpeaks_read, best of 5 reads of a 4 GiB buffer, CUDA events"}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": elapsed_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": workload_config(w) | {"parallelism": f"replicas{world}" if world > 1 else "single",
                                        "l2": flush.note} |
                  ({"serve_loop": {"steps_timed": args.steps, "entries_at_start": n_timed_begin,
                                   "entries_at_end": n_timed_end,
                                   "step": "lookup, then append of the batch's misses (lacache_append_misses)"}}
                   if serve else {}),
        "stage1_kernel": kernel_name,
        "lsh_index": lsh,
        "roofline": roof | {"traffic": traffic, "kernel": f"stage1_{kernel_name}",
                            # a SimHash lookup streams its index and contracts only the admitted pairs
                            "algorithmic_bytes_per_launch": roof.get("algorithmic_index_bytes_per_launch", s1_bytes),
                            "algorithmic_flops_per_launch": None if lsh else flops,
                            "avg_launch_ms": t1_avg_s * 1e3},
        # the exact key check's contraction rate; a SimHash lookup does not perform that contraction
        "tensor": None if lsh else {"achieved_tflops": flops / (elapsed_ms / args.steps / 1e3) / 1e12,
                                    "peak_tflops": peaks["bf16_tflops"],
                                    "frac": flops / (elapsed_ms / args.steps / 1e3) / 1e12 / peaks["bf16_tflops"]},
        "stage_ms": {"stage1": t1_ms / max(1, timed), "stage2": t2_ms / max(1, timed), "timed_lookups": timed},
        "e2e": {"value": job["e2e_value"], "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": args.e2e_steps,
                "api": ("lacache_lookup_host (pinned host buffers, one synchronous call per step, each timed alone "
                        "after an L2 flush)") if flush.on else
                       f"lacache_lookup_host_async (mapped pinned host buffers, {depth} lookups in flight)"},
        "e2e_sync": {"value": sync_job["e2e_value"], "unit": UNIT, "steps": args.e2e_steps,
                     "api": "lacache_lookup_host (pinned host buffers, one synchronous call per step)"},
        "gpu_launches": ((3 if lsh else 2) + (2 if serve else 0)) * args.steps,
        "clocks": clock,
        "decisions": decision_rates(w, batches[0], outs[0]),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w)
    cache.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def decision_rates(w, q: dict, out: dict) -> dict:
    """The paper's hit metrics (section 4.1) on one looked-up batch, from the generator's query classes: the
    benign hit rate (near-duplicates served their own target), the attack hit rate (collision and mimic queries
    served anything), and the attack hit rate a key check alone would give (those with a candidate above tau_c),
    which the lookahead check brings down."""
    import numpy as np

    from paper_2608_01718_gb300 import lacache as L
    from paper_2608_01718_gb300 import workloads as wl
    cls, tgt = q["class"].cpu().numpy(), q["target"].cpu().numpy()
    status, entry = out["status"].cpu().numpy(), out["entry_id"].cpu().numpy()
    n_cand = out["n_cand"].cpu().numpy()
    near = cls == wl.NEAR
    attack = (cls == wl.COLLISION) | (cls == wl.MIMIC)
    rate = lambda m: float(np.mean(m)) if m.size else None
    return {"queries": int(len(cls)), "near_duplicate": int(near.sum()), "attack": int(attack.sum()),
            "benign_hit_rate": rate((status[near] == L.LACACHE_HIT) & (entry[near] == tgt[near])),
            "attack_hit_rate": rate(status[attack] == L.LACACHE_HIT),
            "attack_hit_rate_key_check_only": rate(n_cand[attack] > 0),
            "random_hit_rate": rate(status[cls == wl.RANDOM] == L.LACACHE_HIT)}


def cpu_baseline(w) -> dict:
    """The oracle on the host cores over a bounded sample: as many store rows as take about 15 s of oracle time
    (all of them if fewer), scaled to the full store."""
    probe = min(w.n, 8192)
    store, oq = oracle_sample(w, probe, 0, "cuda")
    per_row = time_oracle(store, oq, w) / probe
    rows = int(min(w.n, max(probe, 15.0 / per_row)))
    store, oq = oracle_sample(w, rows, 0, "cuda")
    t = time_oracle(store, oq, w)
    return {"value": w.batch / (t * w.n / rows), "unit": UNIT, "cores": cpu_threads(), "kind": "oracle",
            "sample": f"oracle lookup of the {w.batch}-query batch against the first {rows} of the {w.n} store rows "
                      f"({t:.1f} s), scaled to the full store by N/rows (the oracle is linear in N)"}


def run_sharded(args, w):
    """Entry-range sharding: rank r holds store rows [N r / world, N (r + 1) / world); every rank looks up the same
    batches; per lookup, the rank's own lookup, one all-gather of the candidate records and the merge
    (paper_2608_01718_gb300.sharded). Strong scaling: the job serves B queries per step whatever the world size."""
    import torch
    import torch.distributed as dist

    from paper_2608_01718_gb300 import build, sharded
    from paper_2608_01718_gb300 import lacache as L
    from paper_2608_01718_gb300 import workloads as wl

    rank, local_rank, world = rank_info()
    torch.cuda.set_device(local_rank)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    build.build()
    a, b = w.n * rank // world, w.n * (rank + 1) // world
    models = len(w.prefix_dims) if w.prefix_dims is not None else 1
    cache = L.LaCache(w.d, w.k, max(1, b - a), w.tau_c, w.tau_a, w.top_c, max_batch=w.batch, device=local_rank,
                      prefix_dims=w.prefix_dims, tau_a_models=w.tau_a_models)
    dtype = L.LACACHE_F32 if w.key_dtype == "f32" else L.LACACHE_BF16
    off = 0
    for ch in wl.iter_store(w, "cuda"):
        n = ch["key"].shape[0]
        lo, hi = max(a, off), min(b, off + n)
        if lo < hi:
            cache.insert(ch["key"][lo - off:hi - off], ch["prefix"][lo - off:hi - off], ch["ids"][lo - off:hi - off],
                         dtype)
        off += n
        del ch
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    stream = torch.cuda.current_stream()
    scratch = L.alloc_result(w.batch, w.top_c, "cuda", candidates=False)

    def local_lookup(q, rec):
        L.lacache_lookup(cache.h, q["emb"], q["prefix"], q["ids"], {**scratch, **rec}, stream)

    def merge(shards, out):
        L.lacache_merge_shards(shards, w.top_c, models, out, stream)

    lk = sharded.ShardedLookup(w.batch, w.top_c, models, a, "cuda", local_lookup, merge)
    nb = args.batches
    batches = [wl.batch(w, step=i, device="cuda") for i in range(nb)]
    outs = [L.alloc_result(w.batch, w.top_c, "cuda", candidates=False, models=models if models > 1 else 0)
            for _ in range(nb)]

    def step(i):
        lk(batches[i % nb], outs[i % nb])

    for i in range(max(3, args.warmup)):
        step(i)
    torch.cuda.synchronize()
    cache.sync()
    flush = L2Flush(max(1, b - a) * w.d * 2, "shard's keys")
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(torch.cuda.current_device())
    clocks.start()
    elapsed_ms = device_steps_ms(step, args.steps, stream, flush)
    if world > 1:
        dist.barrier()
    clock = clocks.stop()
    cache.sync()
    L.lacache_stage_timing(cache.h, args.steps)
    for i in range(args.steps):
        flush()
        step(i)
    t1_ms, t2_ms, timed = L.lacache_stage_times(cache.h)
    L.lacache_stage_timing(cache.h, 0)

    # end to end: pinned host batch -> device, the sharded lookup, the decisions back to pinned host memory
    hq = [{k: batches[i][k].cpu().pin_memory() for k in ("emb", "prefix", "ids")} for i in range(nb)]
    dq = [{k: torch.empty_like(batches[i][k]) for k in ("emb", "prefix", "ids")} for i in range(nb)]
    keys = ("entry_id", "status", "key_score", "prefix_score", "token_matches", "n_cand")
    hout = [{k: torch.empty_like(outs[i][k], device="cpu").pin_memory() for k in keys} for i in range(nb)]

    def e2e_step(i):
        j = i % nb
        for k in dq[j]:
            dq[j][k].copy_(hq[j][k], non_blocking=True)
        lk(dq[j], outs[j])
        for k in keys:
            hout[j][k].copy_(outs[j][k], non_blocking=True)
        stream.synchronize()

    for i in range(max(3, args.warmup)):
        e2e_step(i)
    if world > 1:
        dist.barrier()
    e2e_s = 0.0
    t0 = time.perf_counter()
    for i in range(args.e2e_steps):
        if flush.on:   # each synchronous step timed alone after a finished flush
            flush()
            torch.cuda.synchronize()
            t0 = time.perf_counter()
        e2e_step(i)
        if flush.on:
            e2e_s += time.perf_counter() - t0
    if not flush.on:
        e2e_s = time.perf_counter() - t0
    times = torch.tensor([elapsed_ms, e2e_s], dtype=torch.float64, device="cuda")
    if world > 1:
        dist.all_reduce(times, op=dist.ReduceOp.MAX)
    elapsed_ms, e2e_s = float(times[0]), float(times[1])

    peaks, peak_src = load_peaks()
    local = w.scaled(n=max(1, b - a))
    s1_bytes, _, flops = algorithmic(local, w.batch)
    t1_avg_s = t1_ms / max(1, timed) / 1e3
    ridge = peaks["bf16_tflops"] * 1e12 / (peaks["hbm_gbs"] * 1e9)
    if flops / s1_bytes < ridge:
        roof = {"bound": "hbm", "achieved": s1_bytes / t1_avg_s / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "peak_source": f"{peak_src} (copy bandwidth)"}
    else:
        roof = {"bound": "tensor", "achieved": flops / t1_avg_s / 1e12, "peak": peaks["bf16_tflops"],
                "unit": "TFLOP/s", "peak_source": f"{peak_src} (burst bf16 dense)"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    kernel_name = {L.LACACHE_STAGE1_TENSOR: "tensor", L.LACACHE_STAGE1_TENSOR_PAIR: "tensor-pair",
                   L.LACACHE_STAGE1_STREAM: "stream", L.LACACHE_STAGE1_LSH: "lsh"}[cache.last_launch()[1]]
    line = {
        "metric": METRIC, "value": w.batch * args.steps / (elapsed_ms / 1e3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": elapsed_ms / args.steps,
        "higher_is_better": True, "scaling": "strong", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": workload_config(w) | {"parallelism": f"entry-shards{world}", "shard_entries": b - a,
                                        "l2": flush.note},
        "stage1_kernel": kernel_name,
        "roofline": roof | {"traffic": None, "kernel": f"stage1_{kernel_name} (one shard)",
                            "algorithmic_bytes_per_launch": s1_bytes, "algorithmic_flops_per_launch": flops,
                            "avg_launch_ms": t1_avg_s * 1e3},
        "stage_ms": {"stage1": t1_ms / max(1, timed), "stage2": t2_ms / max(1, timed), "timed_lookups": timed},
        "e2e": {"value": w.batch * args.e2e_steps / e2e_s, "unit": UNIT,
                "h2d_bytes_per_step": w.batch * (2 * w.d + 2 * w.pd + w.k * 4),
                "d2h_bytes_per_step": w.batch * (4 + 1 + 4 + 4 + 4 + 4), "steps": args.e2e_steps,
                "api": "paper_2608_01718_gb300.sharded.ShardedLookup (pinned host buffers, synchronous per step)"},
        "gpu_launches": 3 * args.steps,
        "clocks": clock,
        "decisions": decision_rates(w, batches[0], outs[0]),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w)
    cache.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


CALIBRATION = {"calib-1m": (1 << 20, 1024, 0.6, 10.0, 0.70)}   # pairs, d, paraphrase noise, percentile, cap


def run_calibration(args):
    """Threshold calibration (App. A.2) over n benign pairs: pair similarities + nearest-rank percentile."""
    import torch

    from paper_2608_01718_gb300 import build
    from paper_2608_01718_gb300 import lacache as L
    from paper_2608_01718_gb300 import workloads as wl
    n, d, sigma, pct, cap = CALIBRATION[args.workload]
    build.build()
    x, y = wl.benign_pairs(n, d, sigma, device="cuda")
    sims = torch.empty(n, dtype=torch.float32, device="cuda")
    res = torch.empty(2, dtype=torch.float32, device="cuda")
    ws = torch.empty(L.lacache_calibrate_workspace_bytes(), dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()
    for _ in range(max(3, args.warmup)):
        L.lacache_calibrate(x, y, pct, cap, sims, res, ws, stream)
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        L.lacache_calibrate(x, y, pct, cap, sims, res, ws, stream)
    ev1.record(stream)
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1) / args.steps
    peaks, src = load_peaks()
    bytes_ = 4 * n * d + 4 * n
    line = {"metric": "calibration pairs/s (App. A.2 thresholds)", "value": n / (ms / 1e3), "unit": "pairs/s",
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "dtype": "bf16", "data": "synthetic",
            "config": {"workload": args.workload, "pairs": n, "d": d, "percentile": pct, "cap": cap},
            "roofline": {"bound": "hbm", "achieved": bytes_ / (ms / 1e3) / 1e9, "peak": peaks["hbm_gbs"],
                         "unit": "GB/s", "frac": bytes_ / (ms / 1e3) / 1e9 / peaks["hbm_gbs"],
                         "peak_source": f"{src} (copy bandwidth)"},
            "result": [float(v) for v in res.cpu()], "gpu_launches": 8 * args.steps}
    print(json.dumps(line), flush=True)
    return 0


VERIFY = {"verify-256": (256, 32)}   # queries, draft tokens: the serve loop's batch (serve-2m) and its k


def run_verify(args):
    """Draft verification of the speculative prefix reuse (section 3.3): per query, the number of leading draft
    tokens with P_f >= P_g, -1 for a served query. Synthetic token probabilities (uniform) and statuses (half
    served); one call per step."""
    import torch

    from paper_2608_01718_gb300 import build
    from paper_2608_01718_gb300 import lacache as L
    B, k = VERIFY[args.workload]
    build.build()
    g = torch.Generator(device="cuda").manual_seed(20261205)
    p_target = torch.rand((B, k), generator=g, device="cuda")
    p_draft = torch.rand((B, k), generator=g, device="cuda")
    status = torch.where(torch.rand(B, generator=g, device="cuda") < 0.5, L.LACACHE_HIT,
                         L.LACACHE_REJECT).to(torch.uint8)
    accepted = torch.empty(B, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()
    for _ in range(max(3, args.warmup)):
        L.lacache_verify_draft(p_target, p_draft, status, accepted, stream)
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        L.lacache_verify_draft(p_target, p_draft, status, accepted, stream)
    ev1.record(stream)
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1) / args.steps
    peaks, src = load_peaks()
    bytes_ = 2 * B * k * 4 + B + 4 * B
    acc = accepted.cpu()
    line = {"metric": "draft verifications/s (section 3.3 prefix reuse)", "value": B / (ms / 1e3),
            "unit": "queries/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "dtype": "f32", "data": "synthetic",
            "config": {"workload": args.workload, "queries": B, "draft_tokens": k, "served_fraction": 0.5},
            "roofline": {"bound": "hbm", "achieved": bytes_ / (ms / 1e3) / 1e9, "peak": peaks["hbm_gbs"],
                         "unit": "GB/s", "frac": bytes_ / (ms / 1e3) / 1e9 / peaks["hbm_gbs"],
                         "peak_source": f"{src} (copy bandwidth)",
                         "note": f"{bytes_} bytes a call: bound by launch and memory latency, not bandwidth"},
            "result": {"served": int((acc == -1).sum()), "mean_accepted": float(acc[acc >= 0].float().mean())},
            "gpu_launches": args.steps}
    print(json.dumps(line), flush=True)
    return 0


def main():
    args = parse_args()
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        # one process per GPU: build once here, so the ranks find the library up to date, then start them
        if args.impl == "ours":
            from paper_2608_01718_gb300 import build
            build.build()
        return launch_ranks(args.gpus, sys.argv[1:])
    from paper_2608_01718_gb300 import workloads as wl
    if args.workload in CALIBRATION:
        return run_calibration(args)
    if args.workload in VERIFY:
        return run_verify(args)
    w = wl.WORKLOADS[args.workload]
    if args.entries:
        w = w.scaled(n=args.entries)
    if args.batch:
        w = w.scaled(batch=args.batch)
    if args.impl == "reference":
        return run_reference(args, w)
    if args.mode == "shard":
        return run_sharded(args, w)
    return run_ours(args, w)


if __name__ == "__main__":
    sys.exit(main())
