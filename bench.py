"""Benchmark: ragged causal GQA prefill attention on GB300 (libopattn).

One step = one pass of the whole hot path (one persistent-kernel launch of
opattn over the workload's ragged batch).  The headline workload is the
Llama-3-70B-shaped layer (Hq 64, Hkv 8, d 128, 8 prompts x 4096 tokens).
The decode workloads (--workload decode_*) time the decode kernel
(opattn_decode) instead; it is bound by HBM, so its roofline is reported in
GB/s of algorithmic traffic (q, k, v and o once, plus LSE).

Metric: causal attention TFLOP/s, counting 4 * d * Hq FLOPs per visible
(query, key) pair (2d for QK^T, 2d for PV; masked and skipped work, softmax
and the dense square are not counted); tokens/s and the fraction of the
measured dense BF16 peak are printed beside it.

Arms:
  --impl ours       (default) the CUDA library; `value` is kernel time with
                    inputs resident in HBM, `e2e` goes through the C-ABI
                    one-shot call with pinned host buffers and includes every
                    step's host<->device copies (pipelined over two buffer
                    sets so that copies overlap the neighbouring steps).
  --impl reference  the fp64 CPU oracle on this machine's cores, each step a
                    bounded row sample of the same workload.

Multi-GPU (torchrun, one process per GPU): every rank runs an independent
replica of the workload (the operator shards by sequence or kv head with no
data exchange); timing is the max over ranks, value the sum of all ranks'
work over that time.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "prefill attention TFLOP/s (causal) and prompt tokens/s on 1 GB300; % BF16 peak"
METRIC_DECODE = "decode attention TFLOP/s (causal) and HBM GB/s on 1 GB300; % measured HBM bandwidth"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# ---------------------------------------------------------------- helpers

def visible_pairs(q_lens, k_lens) -> int:
    """Number of (query, key) pairs the bottom-right causal mask leaves visible."""
    total = 0
    for lq, lk in zip(q_lens, k_lens):
        if lq == 0 or lk == 0:
            continue
        i = np.arange(lq, dtype=np.int64)
        total += int(np.clip(i + (lk - lq) + 1, 0, lk).sum())
    return total


def causal_flops(w) -> int:
    return 4 * w.d * w.Hq * visible_pairs(w.q_lens, w.k_lens)


def algorithmic_bytes(w) -> int:
    """Bytes the operator must move at least: q, k, v read once, o and LSE written once."""
    return 2 * w.d * (2 * w.total_q * w.Hq + 2 * w.total_k * w.Hkv) + 4 * w.total_q * w.Hq


def row_flops(w, tokens, heads) -> int:
    """Causal FLOPs of selected output rows (same per-pair count)."""
    seq = np.searchsorted(w.cu_q, tokens, side="right") - 1
    lq = np.asarray(w.q_lens)[seq]
    lk = np.asarray(w.k_lens)[seq]
    i = tokens - w.cu_q[seq]
    n = np.clip(i + (lk - lq) + 1, 0, lk)
    return int(4 * w.d * n.sum())


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return json.load(f), "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def aggregate_over_ranks(elapsed_s: float, work_units: float, dist=None):
    """(max elapsed over ranks, sum of work over ranks); identity without a process group."""
    if dist is None or not dist.is_available() or not dist.is_initialized():
        return elapsed_s, work_units
    import torch
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([elapsed_s], dtype=torch.float64, device=dev)
    u = torch.tensor([work_units], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), float(u.item())


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms while running."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, gpu_selector: str | None):
        self.sel = gpu_selector
        self.proc = None
        self.lines = []

    def start(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200"]
        if self.sel:
            cmd += ["-i", self.sel]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, pw, reasons = [], [], [], set()
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            try:
                pw.append(float(parts[3]))
            except ValueError:
                pass
            for name, val in zip(self.NAMES, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        res = {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
               "samples": len(sm), "sm_mhz_min": min(sm)}
        if pw:
            res["power_w_median"] = statistics.median(pw)
            res["power_w_max"] = max(pw)
        return res


def gpu_selector(torch, dev):
    props = torch.cuda.get_device_properties(dev)
    uuid = getattr(props, "uuid", None)
    if uuid:
        s = str(uuid)
        return s if s.startswith("GPU-") else "GPU-" + s
    return str(dev)


def cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True).stdout
        for line in out.splitlines():
            if line.startswith("Model name"):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return "unknown"


def oracle_sample(w, q, k, v, seconds: float, seed: int = 0):
    """Time the fp64 oracle on random rows of w for about `seconds`; returns a dict."""
    import oracle
    rng = np.random.default_rng(seed)
    threads = oracle.default_threads()
    n = max(8, threads)
    done_flops, done_rows, t_total = 0, 0, 0.0
    while t_total < seconds:
        tok = rng.integers(0, w.total_q, size=n).astype(np.int64)
        hd = rng.integers(0, w.Hq, size=n).astype(np.int32)
        t0 = time.perf_counter()
        oracle.attention_rows(q, k, v, w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale, tok, hd, n_threads=threads)
        dt = time.perf_counter() - t0
        t_total += dt
        done_flops += row_flops(w, tok, hd)
        done_rows += n
        if dt < seconds / 8:
            n *= 2
    return {"flops": done_flops, "seconds": t_total, "rows": done_rows, "threads": threads}


def host_time_us(fn, reps: int, torch, dev) -> float:
    """Median host time of fn() in microseconds, each call made with the GPU idle
    (synchronized before the call; the call itself is not waited for)."""
    ts = []
    for _ in range(reps):
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter_ns()
        fn()
        ts.append((time.perf_counter_ns() - t0) / 1e3)
    torch.cuda.synchronize(dev)
    return statistics.median(ts)


def copy_ceiling(pairs_in, pairs_out, steps: int, flops: int, torch, dev):
    """Rates of the e2e loop's copies alone, one cudaMemcpyAsync per tensor as the loop
    issues them: host->device only, device->host only, and both directions at once on
    two streams.  Returns the dict of the bench line's e2e.copy_ceiling."""
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    b_in = sum(d.numel() * d.element_size() for d, _ in pairs_in)
    b_out = sum(h.numel() * h.element_size() for h, _ in pairs_out)

    def timed(do_in, do_out):
        for _ in range(2):  # warm
            with torch.cuda.stream(s_in):
                for d, h in (pairs_in if do_in else []):
                    d.copy_(h, non_blocking=True)
            with torch.cuda.stream(s_out):
                for h, d in (pairs_out if do_out else []):
                    h.copy_(d, non_blocking=True)
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        cur = torch.cuda.current_stream(dev)
        e0.record(cur)
        s_in.wait_event(e0)
        s_out.wait_event(e0)
        for _ in range(steps):
            with torch.cuda.stream(s_in):
                for d, h in (pairs_in if do_in else []):
                    d.copy_(h, non_blocking=True)
            with torch.cuda.stream(s_out):
                for h, d in (pairs_out if do_out else []):
                    h.copy_(d, non_blocking=True)
        cur.wait_stream(s_in)
        cur.wait_stream(s_out)
        e1.record(cur)
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1) / steps  # ms per step

    ms_in = timed(True, False)
    ms_out = timed(False, True)
    ms_both = timed(True, True)
    return {"steps": steps, "h2d_gbs": b_in / ms_in / 1e6, "d2h_gbs": b_out / ms_out / 1e6,
            "both_ms_per_step": ms_both, "both_gbs": (b_in + b_out) / ms_both / 1e6,
            "ceiling_value": flops / (ms_both / 1e3) / 1e12,
            "how": "the e2e loop's own tensors, one cudaMemcpyAsync per tensor; 'both' runs the H2D and D2H "
                   "streams concurrently, ceiling_value = FLOPs per step / both_ms_per_step"}


# ----------------------------------------------------------- reference arm

REFERENCE_BUDGET_S = 150.0  # host time of the reference arm's timed steps

def run_reference(args, w):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import torch
    from paper_2608_13499_gb300 import workloads as W
    q, k, v = W.make_inputs(w, "cpu")
    qb, kb, vb = q, k, v
    # Each step is a bounded sample; the whole timed run stays within about
    # REFERENCE_BUDGET_S however many steps are asked for.
    per_step = min(args.reference_step_seconds, max(0.05, REFERENCE_BUDGET_S / max(1, args.steps)))
    for _ in range(args.warmup):
        oracle_sample(w, qb, kb, vb, per_step / 4, seed=1)
    flops, secs, rows = 0, 0.0, 0
    for s in range(args.steps):
        r = oracle_sample(w, qb, kb, vb, per_step, seed=100 + s)
        flops += r["flops"]
        secs += r["seconds"]
        rows += r["rows"]
        threads = r["threads"]
    value = flops / secs / 1e12
    tokens_per_s = value * 1e12 / (causal_flops(w) / w.total_q)
    line = {
        "impl": "reference", "metric": METRIC_DECODE if is_decode(w) else METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": secs / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded N(0,1) bf16 inputs; counter-based generator)",
        "config": bench_config(w, args.gpus),
        "tokens_per_s": tokens_per_s,
        "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": threads, "kind": "oracle",
                         "sample": f"{rows} random output rows of {w.name} over {args.steps} steps, "
                                   f"~{per_step:.1f} s each, fp64, {cpu_model()}"},
        "gpu_launches": 0,
    }
    print(json.dumps(line), flush=True)
    return 0


# -------------------------------------------------------------- our arm

def run_ours(args, w):
    import torch
    import torch.distributed as dist

    import paper_2608_13499_gb300 as pkg
    from paper_2608_13499_gb300 import build as pbuild
    from paper_2608_13499_gb300 import workloads as W

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world != args.gpus:
        raise SystemExit(f"--gpus {args.gpus} but WORLD_SIZE={world}: launch N>1 with torchrun")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    if rank == 0 or world == 1:
        pbuild.build()
    if world > 1:
        dist.barrier()
    pkg.load()

    peaks, peak_src = load_peaks()
    q, k, v = W.make_inputs(w, dev)
    o = torch.empty((w.total_q, w.Hq, w.d), dtype=torch.bfloat16, device=dev)
    lse = torch.empty((w.total_q, w.Hq), dtype=torch.float32, device=dev)
    flops = causal_flops(w)
    stream = torch.cuda.current_stream(dev)

    decode = is_decode(w)
    paged = w.page_size > 0
    if paged:
        # K/V live in a paged cache (shuffled pages); the packed copies are only the source.
        lay = W.paged_layout(w.k_lens, w.page_size, seed=w.seed)
        k_packed, v_packed = k, v
        k, v = W.to_paged(k, w.k_lens, lay), W.to_paged(v, w.k_lens, lay)
        table = torch.from_numpy(lay.block_table).to(dev)
        seqlens_k = np.asarray(w.k_lens, dtype=np.int32)
        plan = pkg.Plan(w.cu_q, seqlens_k, w.Hq, w.Hkv, w.d, decode=True, block_size=w.page_size,
                        max_blocks=lay.max_blocks)

        def run_plan():
            plan.run_paged(q, k, v, table, lay.num_blocks, o, lse, w.scale, stream)

        def one_shot(dq, dk, dv, do, dl):
            pkg.opattn_decode_paged(dq, dk, dv, table, lay.num_blocks, lay.page_size, lay.max_blocks, do, dl,
                                    w.cu_q, seqlens_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale, stream)
    else:
        plan = pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, decode=decode)
        call = pkg.opattn_decode if decode else pkg.opattn_prefill

        def run_plan():
            plan.run(q, k, v, o, lse, w.scale, stream)

        def one_shot(dq, dk, dv, do, dl):
            call(dq, dk, dv, do, dl, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale, stream)
    for _ in range(max(args.warmup, 3)):
        run_plan()
    torch.cuda.synchronize(dev)

    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    sampler = ClockSampler(gpu_selector(torch, local))
    sampler.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for i in range(args.steps):
        ev[i][0].record(stream)
        run_plan()
        ev[i][1].record(stream)
    t_end.record(stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    elapsed = t_start.elapsed_time(t_end) / 1e3
    launch_ms = [a.elapsed_time(b) for a, b in ev]
    elapsed_max, flops_all = aggregate_over_ranks(elapsed, float(flops) * args.steps, dist if world > 1 else None)
    value = flops_all / elapsed_max / 1e12
    kernel_ms = statistics.mean(launch_ms)
    achieved = flops / (kernel_ms / 1e3) / 1e12

    # Sustained: back-to-back plan runs for a fixed duration (the board settles at its
    # power cap), with the clocks sampled over that stretch; compared with the measured
    # sustained GEMM peak.
    sustained = None
    if args.sustained_seconds > 0:
        n_sus = max(args.steps, int(math.ceil(args.sustained_seconds / (kernel_ms / 1e3))))
        sampler2 = ClockSampler(gpu_selector(torch, local))
        sampler2.start()
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        for _ in range(n_sus):
            run_plan()
        s1.record(stream)
        torch.cuda.synchronize(dev)
        clocks_sus = sampler2.stop()
        sus_s, sus_flops = aggregate_over_ranks(s0.elapsed_time(s1) / 1e3, float(flops) * n_sus,
                                                dist if world > 1 else None)
        sustained = {"launches": n_sus, "seconds": sus_s, "value": sus_flops / sus_s / 1e12, "unit": "TFLOP/s",
                     "clocks": clocks_sus}

    # End to end through the one-shot C-ABI call with pinned host buffers.  Every
    # step copies its inputs host -> device, runs the call and copies O and LSE
    # back, all inside the timed region.  Three device buffer sets and separate
    # copy streams let step i + 1's input copy and step i - 1's output copy run
    # while step i computes, as a serving loop that stages the next batch would.
    # As many steps as the device-timed region and at least 100 (unless
    # --e2e-steps sets the count), so that the pipeline's fill (the first
    # step's input copy) and drain (the last step's output copy) weigh as
    # little as they do in a serving loop.
    e2e_steps = max(3, args.e2e_steps) if args.e2e_steps > 0 else max(args.steps, 100)
    hq = q.cpu().pin_memory()
    hk = k.cpu().pin_memory()
    hv = v.cpu().pin_memory()
    slots = 3
    ho = [torch.empty(o.shape, dtype=o.dtype).pin_memory() for _ in range(slots)]
    hl = [torch.empty(lse.shape, dtype=lse.dtype).pin_memory() for _ in range(slots)]
    dq = [torch.empty_like(q) for _ in range(slots)]
    dk = [torch.empty_like(k) for _ in range(slots)]
    dv = [torch.empty_like(v) for _ in range(slots)]
    do = [torch.empty_like(o) for _ in range(slots)]
    dl = [torch.empty_like(lse) for _ in range(slots)]
    h2d_stream, d2h_stream = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    in_ready = [torch.cuda.Event() for _ in range(slots)]
    computed = [torch.cuda.Event() for _ in range(slots)]
    copied_out = [torch.cuda.Event() for _ in range(slots)]

    def e2e_step(i):
        sl = i % slots
        with torch.cuda.stream(h2d_stream):
            h2d_stream.wait_event(computed[sl])          # the slot's inputs are free again
            dq[sl].copy_(hq, non_blocking=True)
            dk[sl].copy_(hk, non_blocking=True)
            dv[sl].copy_(hv, non_blocking=True)
            in_ready[sl].record(h2d_stream)
        stream.wait_event(in_ready[sl])
        stream.wait_event(copied_out[sl])                 # the slot's outputs were read back
        one_shot(dq[sl], dk[sl], dv[sl], do[sl], dl[sl])
        computed[sl].record(stream)
        with torch.cuda.stream(d2h_stream):
            d2h_stream.wait_event(computed[sl])
            ho[sl].copy_(do[sl], non_blocking=True)
            hl[sl].copy_(dl[sl], non_blocking=True)
            copied_out[sl].record(d2h_stream)

    def e2e_run(n):
        for i in range(n):
            e2e_step(i)
        stream.wait_stream(d2h_stream)

    # warm every buffer set and the library's pinned staging pool before timing
    e2e_run(2 * slots)
    torch.cuda.synchronize(dev)
    # The host link's throughput drifts over minutes on a shared machine, so its
    # ceiling is measured right before and right after the e2e loop.
    ceil_steps = min(e2e_steps, 50)
    ceiling_before = copy_ceiling([(dq[0], hq), (dk[0], hk), (dv[0], hv)], [(ho[0], do[0]), (hl[0], dl[0])],
                                  ceil_steps, flops, torch, dev)
    if world > 1:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    h2d_stream.wait_event(e0)
    d2h_stream.wait_event(e0)
    e2e_run(e2e_steps)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    e2e_elapsed, e2e_flops = aggregate_over_ranks(e0.elapsed_time(e1) / 1e3, float(flops) * e2e_steps,
                                                  dist if world > 1 else None)
    e2e_value = e2e_flops / e2e_elapsed / 1e12
    h2d = q.numel() * 2 + k.numel() * 2 + v.numel() * 2  # for a paged cache: the whole cache
    d2h = o.numel() * 2 + lse.numel() * 4
    ceiling_after = copy_ceiling([(dq[0], hq), (dk[0], hk), (dv[0], hv)], [(ho[0], do[0]), (hl[0], dl[0])],
                                 ceil_steps, flops, torch, dev)
    ceiling = {"before": ceiling_before, "after": ceiling_after,
               "ceiling_value": 0.5 * (ceiling_before["ceiling_value"] + ceiling_after["ceiling_value"])}
    ceiling["e2e_over_ceiling"] = e2e_value / ceiling["ceiling_value"]

    # Host time of the one-shot call (validation, schedule, staging, launches) with the GPU
    # idle, beside the scheduler alone and the cost of a ctypes call that does nothing.
    lib = pkg.load()
    host = None
    if not paged:
        cq_np = np.ascontiguousarray(w.cu_q, dtype=np.int32)
        ck_np = np.ascontiguousarray(w.cu_k, dtype=np.int32)
        cq_p, ck_p = cq_np.ctypes.data, ck_np.ctypes.data
        entry = lib.opattn_decode if decode else lib.opattn_prefill
        raw_args = (dq[0].data_ptr(), dk[0].data_ptr(), dv[0].data_ptr(), do[0].data_ptr(), dl[0].data_ptr(),
                    cq_p, ck_p, w.n_seq, w.Hq, w.Hkv, w.d, w.scale, stream.cuda_stream)
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        n_units_c, n_used_c = ctypes.c_int64(0), ctypes.c_int32(0)
        sched = lib.opattn_decode_schedule_default if decode else lib.opattn_schedule
        sched(cq_p, ck_p, w.n_seq, w.Hq, w.Hkv, w.d, sms, None, 0, None, ctypes.byref(n_units_c),
              ctypes.byref(n_used_c))
        width = len(pkg.DEC_UNIT_FIELDS if decode else pkg.UNIT_FIELDS)
        u_buf = np.zeros((max(1, n_units_c.value), width), dtype=np.int32)
        o_buf = np.zeros(sms + 1, dtype=np.int32)
        u_p, o_p = u_buf.ctypes.data, o_buf.ctypes.data
        host = {
            "us_per_call": host_time_us(lambda: entry(*raw_args), 60, torch, dev),
            "schedule_us": host_time_us(lambda: sched(cq_p, ck_p, w.n_seq, w.Hq, w.Hkv, w.d, sms, u_p,
                                                      u_buf.shape[0], o_p, ctypes.byref(n_units_c),
                                                      ctypes.byref(n_used_c)), 60, torch, dev),
            "ffi_us": host_time_us(lib.opattn_version, 60, torch, dev),
            "kernel_us": kernel_ms * 1e3,
            "how": "median of 60 calls with the GPU idle: us_per_call = the one-shot C call (validation, "
                   "schedule, staging, upload and attention launches); schedule_us = the host scheduler "
                   "alone; ffi_us = a ctypes call that does nothing",
        }
    plan.close()

    cpu_base = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        qc, kc, vc = (hq, hk, hv) if not paged else (hq, k_packed.cpu(), v_packed.cpu())
        r = oracle_sample(w, qc, kc, vc, args.cpu_seconds)
        cpu_base = {"value": r["flops"] / r["seconds"] / 1e12, "unit": "TFLOP/s", "cores": r["threads"],
                    "kind": "oracle",
                    "sample": f"{r['rows']} random output rows of {w.name} (fp64 oracle, {r['seconds']:.1f} s, "
                              f"{cpu_model()})"}

    if rank == 0:
        peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
        peak_sus = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
        traffic = recorded_traffic(w.name, decode)
        if decode:
            hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
            gbs = algorithmic_bytes(w) / (kernel_ms / 1e3) / 1e9
            roofline = {"bound": "hbm", "achieved": gbs, "peak": hbm, "unit": "GB/s", "frac": gbs / hbm,
                        "traffic": traffic, "algorithmic_bytes": algorithmic_bytes(w),
                        "peak_source": f"{peak_src} hbm_gbs"}
        else:
            roofline = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                        "frac": achieved / peak, "traffic": traffic,
                        "peak_source": f"{peak_src} bf16_tflops (burst)"}
        line = {
            "metric": METRIC_DECODE if decode else METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
            "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": elapsed_max / args.steps * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded N(0,1) bf16 q/k/v from a counter-based generator)",
            "config": bench_config(w, world),
            "tokens_per_s": value * 1e12 / (flops / w.total_q),
            "pct_bf16_peak": value / peak,
            "pct_bf16_peak_sustained": value / peak_sus,
            "kernel_ms": kernel_ms,
            "flops_per_step": flops,
            "roofline": roofline,
            "e2e": {"value": e2e_value, "unit": "TFLOP/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "steps": e2e_steps, "pipelined": "three buffer sets; copies overlap the neighbouring steps",
                    "gpu_launches": 2 * e2e_steps,  # per one-shot call: the work-list upload and the attention kernel
                    "copy_ceiling": ceiling},
            "host_us_per_call": host["us_per_call"] if host else None,
            "host": host,
            "sustained": (dict(sustained, frac=sustained["value"] / peak_sus,
                               peak=peak_sus, peak_source=f"{peak_src} bf16_tflops_sustained")
                          if sustained and not decode else sustained),
            "cpu_baseline": cpu_base,
            "clocks": clocks,
            "gpu_launches": args.steps,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def bench_config(w, world: int) -> dict:
    """The workload description both arms print as `config` (the same dict, so the two lines compare)."""
    return dict(w.describe(), parallelism=f"replicas{world}" if world > 1 else "single_gpu",
                l2="inputs larger than L2 (q+k+v+o of the workload exceed the 129 MB L2)")


def is_decode(w) -> bool:
    from paper_2608_13499_gb300 import workloads as W
    return any(f().name == w.name for f in W.DECODE.values())


def recorded_traffic(workload: str, decode: bool = False):
    """DRAM bytes per launch from the committed ncu record, or None when the
    kernel sources changed since that capture (the counters no longer apply)."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    rev = kernel_revision(decode)
    with open(path) as f:
        for line in f:
            parts = line.split()
            if len(parts) == 3 and not line.startswith("#") and parts[0] == workload and parts[1] == rev:
                return int(parts[2])
    return None


def kernel_revision(decode: bool = False) -> str:
    """Hash of the kernel and scheduler sources: traffic counters are only valid for the kernel and
    the work order they were taken on."""
    import hashlib
    h = hashlib.sha1()
    for f in ("opattn_decode.cu" if decode else "opattn_kernel.cu", "device_common.cuh", "ptx.cuh",
              "opattn_internal.h", "opattn_api.cpp"):
        with open(os.path.join(ROOT, "paper_2608_13499_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:12]


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="llama3_70b",
                    help="tiny | llama3_8b | llama3_70b | bursty | chunked | chunk_long_prefix | "
                         "chunks_long_prefix | decode_llama3_70b | "
                         "decode_llama3_8b | decode_spec4_llama3_70b | decode_llama3_70b_paged16")
    ap.add_argument("--e2e-steps", type=int, default=0,
                    help="steps of the end-to-end measurement (default 0: as many as --steps, at least 100)")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--sustained-seconds", type=float, default=3.0,
                    help="duration of the back-to-back 'sustained' measurement (0: skip)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--reference-step-seconds", type=float, default=3.0,
                    help="oracle time per reference step, capped so that all steps take about "
                         f"{REFERENCE_BUDGET_S:.0f} s")
    args = ap.parse_args(argv)
    from paper_2608_13499_gb300 import workloads as W
    w = {**W.STANDARD, **W.LONG_PREFIX, **W.DECODE}[args.workload]()
    if args.impl == "reference":
        return run_reference(args, w)
    return run_ours(args, w)


if __name__ == "__main__":
    sys.exit(main())
