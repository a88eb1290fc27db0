"""Benchmark: audio-seconds processed per second through the whole hot path
(append + chunked-prefill and decode attention of every layer + eviction), on
the 64-session ten-minute workload (32 layers, 32/8 heads, head_dim 128, bf16,
B=4096, W=10, session starts U{0..300} s).

One step advances every active session by one one-second unit.  The cache is
first brought (untimed, append + evict only: attention changes no state) to
the step where every session is active and at its budget; W warm-up steps
follow, then K timed steps.  Per-step K/V traffic is hundreds of GB, far
above the 129 MB L2, so no flush is needed between steps.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  N > 1 (torchrun): every rank runs an
independent replica of the workload (sessions are independent; no
collective on the data path): weak scaling.
"""
from __future__ import annotations

import argparse
import hashlib
import re
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "audio-seconds processed/sec (evict+attn, all layers); HBM GB/s vs GB300 peak"
UNIT = "audio-s/s"


# DRAM bytes per algorithmic byte of the roofline kernel (reads + writes), from one
# ncu capture of the stream-K kernel on the 64-session, two-layer case (the bench's
# launch shape; smaller calls run the pair-split kernel): 1,088.57 MB of traffic
# (1,084.41 MB read, 4.16 MB written) for a 1,077.10 MB launch.  Valid only while the
# decode sources hash to the version it was taken on; the roofline's traffic is null
# otherwise.
DECODE_TRAFFIC_RATIO = 1088.57 / 1077.10
DECODE_TRAFFIC_SOURCES = ("paper_2609_31224_gb300/csrc/kvc_attn_decode.cu",
                          "paper_2609_31224_gb300/csrc/kvc_decode_common.cuh",
                          "paper_2609_31224_gb300/csrc/kvc_internal.cuh")
DECODE_TRAFFIC_SHA256 = "1e7582c380f739e8b63919fc568b9687161723d1076652b086603f3e9759a8e7"


def code_only(text: str) -> str:
    """C/C++ source without its comments and with whitespace collapsed: what the compiler
    sees of it (the decode sources hold no string literal with a comment marker)."""
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def decode_sources_digest(root: str | None = None) -> str:
    """SHA-256 of the decode sources' code (comments and layout excluded)."""
    h = hashlib.sha256()
    for f in DECODE_TRAFFIC_SOURCES:
        with open(os.path.join(root or ROOT, f), encoding="utf-8") as fh:
            h.update(code_only(fh.read()).encode())
    return h.hexdigest()


def decode_traffic(alg_bytes_per_launch):
    """Per-launch DRAM traffic of the decode kernel, scaled from the capture, or None."""
    if not alg_bytes_per_launch:
        return None
    if decode_sources_digest() != DECODE_TRAFFIC_SHA256:
        return None
    return DECODE_TRAFFIC_RATIO * alg_bytes_per_launch


def decode_kernel_label(w) -> str:
    """Kernel that the library's dispatch gives a full-batch decode call of `w` (sessions
    at full budget): the 16-warp pair split while every (session, KV head) pair gets five
    one-CTA-per-SM slices, the 4-warp pair split while it gets one of the three CTAs per
    SM, else stream-K."""
    import torch
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    pairs = w.n_sessions * w.kv_heads
    if 5 * pairs <= sms:
        return "attn_decode_split_kernel (16 warps)"
    if pairs <= 3 * sms:
        return "attn_decode_split_kernel (4 warps)"
    return "attn_decode_kernel"


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# -- clocks sampled during the timed region ------------------------------------------------
class Clocks:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax),
                "samples": len(sm), "reasons": sorted(reasons)}


# -- algorithmic bytes -------------------------------------------------------------------------
def step_bytes(w, drv, st, prev_resident: dict) -> tuple[float, float, int]:
    """(attention+append bytes of the step, bytes of its first full-batch decode round per
    layer launch, number of decode sessions in that round)."""
    esz = 2 if w.dtype == "bf16" else 4
    per_pos_layer = w.kv_heads * w.head_dim * 2 * esz           # K+V of one position, one layer
    q_row = w.q_heads * w.head_dim * esz
    total = 0.0
    n_now = {s: prev_resident.get(s, 0) for s, _ in st.pairs}
    round0_bytes, round0_n = 0.0, 0
    dec_round = 0
    for c in st.calls:
        cnt = np.diff(c.cu)
        for s, t in zip(c.sessions.tolist(), cnt.tolist()):
            n_now[s] += t
        total += int(c.cu[-1]) * w.layers * per_pos_layer        # append: K+V written
        if c.kind == "prefix":
            continue
        keys = sum(n_now[s] for s in c.sessions.tolist())
        per_launch = keys * per_pos_layer + 2 * int(c.cu[-1]) * q_row
        total += w.layers * per_launch
        if c.kind == "decode":
            if dec_round == 0:
                round0_bytes, round0_n = per_launch, len(c.sessions)
            dec_round += 1
    return total, round0_bytes, round0_n


def job_throughput(units: float, elapsed_ms: float, world: int) -> tuple[float, float]:
    """Whole-job throughput: the units all ranks processed over the slowest rank's time.
    Returns (units per second, max elapsed ms).  With world > 1 it reduces over the
    default process group (NCCL: CUDA tensors, gloo: host tensors)."""
    if world > 1:
        import torch
        import torch.distributed as dist
        dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
        u = torch.tensor([float(units)], dtype=torch.float64, device=dev)
        t = torch.tensor([float(elapsed_ms)], dtype=torch.float64, device=dev)
        dist.all_reduce(u, op=dist.ReduceOp.SUM)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        units, elapsed_ms = float(u.item()), float(t.item())
    return units / (elapsed_ms / 1e3), elapsed_ms


def workload_config(w, start: int, steps: int, world: int, per_layer: bool) -> dict:
    """The `config` object of the JSON line (both arms)."""
    return {
        "workload": w.name,
        "sessions": w.n_sessions, "layers": w.layers, "q_heads": w.q_heads,
        "kv_heads": w.kv_heads, "head_dim": w.head_dim, "page_size": w.page_size,
        "budget": w.budget, "window": w.window, "units_per_session": w.units,
        "offsets": f"U{{0..{w.offset_max}}}", "timed_steps": [start, start + steps],
        "l2": "no flush: per-step K/V traffic >> 129 MB L2",
        "parallelism": f"replicas x{world}",
        "append": "per-layer" if per_layer else "whole chunk",
    }


def run_ours(args, rank: int, world: int, local_rank: int):
    import torch
    from synth import script as S
    from synth.driver import Driver

    torch.cuda.set_device(local_rank)
    w = S.BATCH64_BF16
    if args.sessions or args.layers:
        # Reduced case of the same kernels (for profiler captures that must stay small).
        w = w.with_(n_sessions=args.sessions or w.n_sessions, layers=args.layers or w.layers,
                    name=f"{w.name}-reduced-{args.sessions or w.n_sessions}s-"
                         f"{args.layers or w.layers}L")
    scripts = S.workload_scripts(w)
    drv = Driver(w, scripts)
    start = args.start if args.start is not None else S.steady_state_step(w, scripts)
    n_steps_total = len(drv.sched)
    assert start - args.warmup >= 0 and start + args.steps <= n_steps_total
    # The end-to-end run covers the timed steps again (from a second cache in the same
    # state): step cost varies with the decode rounds (speaking turns), so other steps
    # would not be comparable.
    e2e_steps = args.e2e_steps if args.e2e_steps is not None else args.steps
    assert start + e2e_steps <= n_steps_total

    # 1. Bring the cache to the step before the warm-up (append + evict only).
    drv.fast_forward(start - args.warmup)
    torch.cuda.synchronize()

    # 2. Inputs of the warm-up and timed steps, resident on the device.
    warm = [drv.prepare_step() for _ in range(args.warmup)]
    timed = [drv.prepare_step() for _ in range(args.steps)]
    n_res_buf = torch.zeros((args.steps + 1, w.n_sessions), dtype=torch.int64, device="cuda")
    stream = torch.cuda.current_stream()

    idx_of = {id(st): torch.as_tensor(st.evict_sessions.astype(np.int64), device="cuda")
              for st in warm + timed}

    def snapshot_resident(row, st):
        idx = idx_of[id(st)]
        n_res_buf[row].index_copy_(0, idx, drv.resident_out[:len(idx)])

    for st in warm:
        drv.run_step(st)
    snapshot_resident(0, warm[-1])
    torch.cuda.synchronize()

    # 3. Timed steps.  Events around the first full-batch decode round (all layers) of every
    #    step give the decode kernel's live per-launch duration.
    dec_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in timed]
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    launches = 0
    clocks = Clocks(local_rank)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clocks.start()
    torch.cuda.nvtx.range_push("timed")
    host0 = time.perf_counter()
    t0.record(stream)
    per_layer = args.per_layer_append
    for i, st in enumerate(timed):
        first_dec = next((c for c in st.calls if c.kind == "decode"), None)
        for c in st.calls:
            if c is first_dec and not per_layer:
                _, s_p, _, c_p, t_ptr, k_ptr, v_ptr, q_ptrs, o_ptr = c.raw
                drv.cache.append_chunk_raw(len(c.sessions), s_p, c_p, t_ptr, k_ptr, v_ptr,
                                           drv.stream)
                dec_ev[i][0].record(stream)
                for layer in range(w.layers):
                    drv.cache.attn_decode_raw(layer, q_ptrs[layer], o_ptr, drv.stream)
                dec_ev[i][1].record(stream)
                launches += 2 + w.layers
            elif c is first_dec:
                # The model's order: each layer's K/V written by its own decode launch
                # (fused); each launch is timed on its own.
                _, s_p, _, c_p, t_ptr, k_ptr, v_ptr, q_ptrs, o_ptr = c.raw
                drv.cache.append_chunk_raw(len(c.sessions), s_p, c_p, t_ptr, None, None,
                                           drv.stream)
                kv_stride = c.k.stride(0) * c.k.element_size()
                evs = []
                for layer in range(w.layers):
                    e0 = torch.cuda.Event(enable_timing=True)
                    e1 = torch.cuda.Event(enable_timing=True)
                    e0.record(stream)
                    drv.cache.attn_decode_kv_raw(layer, k_ptr + layer * kv_stride,
                                                 v_ptr + layer * kv_stride, q_ptrs[layer], o_ptr,
                                                 drv.stream)
                    e1.record(stream)
                    evs.append((e0, e1))
                dec_ev[i] = evs
                launches += 1 + w.layers
            else:
                launches += drv.run_call(c, per_layer=per_layer)
        drv.cache.evict(st.evict_sessions, drv.resident_out)
        launches += 2
        snapshot_resident(i + 1, st)
    t1.record(stream)
    host_submit_s = time.perf_counter() - host0
    torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    clk = clocks.stop()
    audio_s = sum(len(st.pairs) for st in timed)          # one unit = one audio second
    value, elapsed_ms = job_throughput(audio_s, t0.elapsed_time(t1), world)

    # Algorithmic bytes (attention reads every resident K/V byte once per call per layer).
    res = n_res_buf.cpu().numpy()
    tot_bytes, dec_bytes, dec_times = 0.0, [], []
    for i, st in enumerate(timed):
        prev = {s: int(res[i, s]) for s, _ in st.pairs}
        b, rb, _ = step_bytes(w, drv, st, prev)
        tot_bytes += b
        if rb:
            dec_bytes.append(rb)
            ev = dec_ev[i]
            dec_times.append(sum(a.elapsed_time(b) for a, b in ev) / len(ev) if isinstance(ev, list)
                             else ev[0].elapsed_time(ev[1]) / w.layers)
    del timed, warm, idx_of, snapshot_resident, n_res_buf, drv
    torch.cuda.synchronize()
    torch.cuda.empty_cache()

    # 4. End to end through the public API over the same steps: a second cache (the first
    #    one released) brought to the same state and warmed up the same way; then every
    #    step's inputs are copied from pinned host memory and its results (every call's
    #    output, resident counts) read back inside the timed region.
    drv = Driver(w, scripts)
    drv.fast_forward(start - args.warmup)
    for _ in range(args.warmup):
        drv.run_step(drv.prepare_step())
    torch.cuda.synchronize()
    e2e = run_e2e(drv, w, e2e_steps, world, args.per_layer_append)
    del drv
    torch.cuda.empty_cache()

    peak, peak_kind = load_peaks()
    dec_gbs = (sum(dec_bytes) / 1e9) / (sum(dec_times) / 1e3) if dec_times else None
    out = {
        "metric": METRIC,
        "value": value,
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": elapsed_ms / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": w.dtype,
        "data": "synthetic (seeded SplitMix64 Irwin-Hall values, PCG64 session scripts)",
        "config": dict(workload_config(w, start, args.steps, world, args.per_layer_append),
                       audio_seconds_timed_per_gpu=audio_s),
        "path_hbm_gbs": (tot_bytes / 1e9) / (elapsed_ms / 1e3),
        "path_frac_of_peak": (tot_bytes / 1e9) / (elapsed_ms / 1e3) / peak,
        "roofline": {
            "kernel": decode_kernel_label(w),
            "bound": "hbm",
            "achieved": dec_gbs,
            "peak": peak,
            "peak_kind": f"{peak_kind} copy bandwidth",
            "unit": "GB/s",
            "frac": (dec_gbs / peak) if dec_gbs else None,
            "traffic": decode_traffic((sum(dec_bytes) / len(dec_bytes)) if dec_bytes else None),
            "traffic_note": "ncu DRAM bytes per algorithmic byte of the stream-K kernel on "
                            "the 64-session two-layer case, times this launch's bytes",
            "algorithmic_bytes_per_launch": (sum(dec_bytes) / len(dec_bytes)) if dec_bytes else None,
            "avg_launch_us": (1e3 * sum(dec_times) / len(dec_times)) if dec_times else None,
        },
        "e2e": e2e,
        "gpu_launches": launches,
        "host_submit_ms_per_step": 1e3 * host_submit_s / args.steps,
        "clocks": clk,
    }
    return out


def run_e2e(drv, w, n_steps: int, world: int, per_layer: bool = False) -> dict:
    import torch
    stream = torch.cuda.current_stream()
    first_step = drv.step_index
    steps = [drv.prepare_step() for _ in range(n_steps)]
    # Move every input to pinned host memory; keep same-shaped device buffers.
    host, dev = [], []
    for st in steps:
        hs, ds = [], []
        for c in st.calls:
            names = ["types", "k", "v"] + (["q"] if c.q is not None else [])
            h = {n: getattr(c, n).cpu().pin_memory() for n in names}
            hs.append(h)
            ds.append({n: getattr(c, n) for n in names})
        host.append(hs)
        dev.append(ds)
    res_host = torch.empty(w.n_sessions, dtype=torch.int64).pin_memory()
    # One resident-count buffer per step: a step's evict never overwrites counts that
    # the result stream has not copied yet.
    res_dev = torch.zeros((n_steps, w.n_sessions), dtype=torch.int64, device="cuda")
    out_host = [[torch.empty(c.out.shape, dtype=c.out.dtype).pin_memory() if c.out is not None
                 else None for c in st.calls] for st in steps]
    h2d = sum(t.numel() * t.element_size() for hs in host[0] for t in hs.values())
    d2h = res_host.numel() * 8 + sum(o.numel() * o.element_size()
                                     for o in out_host[0] if o is not None)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    # Inputs move on a copy stream, AHEAD steps ahead of the compute: step i+AHEAD's copies
    # are enqueued just before step i's launches, and each step's compute waits only for
    # its own inputs, so transfers overlap earlier steps' compute (the host runs at most a
    # bounded number of launches ahead of the device, so copies enqueued one step ahead can
    # start too late on a slow host link).  Results come back on a third stream, each
    # after an event behind the call that wrote it, so the compute stream never queues
    # behind a copy.
    AHEAD = 2
    copy_stream = torch.cuda.Stream()
    d2h_stream = torch.cuda.Stream()
    copy_start = [torch.cuda.Event(enable_timing=True) for _ in steps]
    comp = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for _ in steps]
    ready = [torch.cuda.Event(enable_timing=True) for _ in steps]
    t0 = time.perf_counter()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    copy_stream.wait_stream(stream)
    d2h_stream.wait_stream(stream)
    h2d_total, d2h_total = 0, 0

    def enqueue_copies(si):
        nonlocal h2d_total
        with torch.cuda.stream(copy_stream):
            copy_start[si].record(copy_stream)
            for ci in range(len(steps[si].calls)):
                for n, t in host[si][ci].items():
                    dev[si][ci][n].copy_(t, non_blocking=True)
                    h2d_total += t.numel() * t.element_size()
            ready[si].record(copy_stream)

    for si in range(min(AHEAD, len(steps))):
        enqueue_copies(si)
    for si, st in enumerate(steps):
        if si + AHEAD < len(steps):
            enqueue_copies(si + AHEAD)
        stream.wait_event(ready[si])
        comp[si][0].record(stream)
        for ci, c in enumerate(st.calls):
            drv.run_call(c, per_layer=per_layer)
            if c.out is not None:
                d2h_stream.wait_stream(stream)
                with torch.cuda.stream(d2h_stream):
                    out_host[si][ci].copy_(c.out, non_blocking=True)
                d2h_total += c.out.numel() * c.out.element_size()
        drv.cache.evict(st.evict_sessions, res_dev[si])
        n = len(st.evict_sessions)
        d2h_stream.wait_stream(stream)
        with torch.cuda.stream(d2h_stream):
            res_host[:n].copy_(res_dev[si, :n], non_blocking=True)
        d2h_total += n * 8
        comp[si][1].record(stream)
    stream.wait_stream(d2h_stream)
    e1.record(stream)
    submit = time.perf_counter() - t0
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    wall = time.perf_counter() - t0
    copy_ms = [a.elapsed_time(b) for a, b in zip(copy_start, ready)]
    comp_ms = [a.elapsed_time(b) for a, b in comp]
    audio_s = sum(len(st.pairs) for st in steps)
    value, ms = job_throughput(audio_s, ms, world)
    return {"value": value, "unit": UNIT,
            "h2d_bytes_per_step": h2d_total / n_steps, "d2h_bytes_per_step": d2h_total / n_steps,
            "steps": n_steps, "first_step": first_step, "host_wall_s": wall,
            "host_submit_ms_per_step": 1e3 * submit / n_steps,
            "h2d_ms_per_step": sum(copy_ms) / n_steps,
            "compute_ms_per_step": sum(comp_ms) / n_steps,
            "h2d_gbs": (h2d_total / 1e9) / (sum(copy_ms) / 1e3) if sum(copy_ms) > 0 else None}


# -- budget versus no budget on one session ---------------------------------------------------
def run_unbounded_comparison() -> dict:
    """The single-session workload with B = 4096 and with B = infinity, on the same seeded
    inputs, through all 600 units: peak resident positions and K/V bytes, and the summed
    GPU time of every attention call (events from the end of each call's append to its
    last layer)."""
    import torch
    from synth import script as S
    from synth.driver import Driver
    res = {}
    clocks = Clocks(torch.cuda.current_device())
    clocks.start()
    for w in (S.SINGLE_BF16, S.SINGLE_BF16_UNBOUNDED):
        scripts = S.workload_scripts(w)
        drv = Driver(w, scripts)
        spans = []
        for _ in range(len(drv.sched)):
            st = drv.prepare_step()
            for c in st.calls:
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                drv.run_call(c, on_append=lambda _c, e=e0: e.record())
                e1.record()
                if c.kind != "prefix":
                    spans.append((e0, e1))
            drv.cache.evict(st.evict_sessions, drv.resident_out)
            del st
        torch.cuda.synchronize()
        info = drv.cache.export_state(0)
        res[w.name] = {
            "budget": w.budget,
            "attention_ms": sum(a.elapsed_time(b) for a, b in spans),
            "attention_calls": len(spans) * w.layers,
            "peak_resident_positions": info["peak_resident"],
            "end_resident_positions": info["resident"],
            "peak_kv_bytes": info["peak_resident"] * w.kv_bytes_per_position,
        }
        del drv
        torch.cuda.empty_cache()
    clk = clocks.stop()
    b, f = res[S.SINGLE_BF16.name], res[S.SINGLE_BF16_UNBOUNDED.name]
    return {"comparison": "single session, B=4096 vs B=infinity, same seeded inputs",
            "clocks": clk,
            "units": S.SINGLE_BF16.units, "runs": res,
            "peak_kv_reduction": 1.0 - b["peak_kv_bytes"] / f["peak_kv_bytes"],
            "attention_time_ratio_full_over_budget": f["attention_ms"] / b["attention_ms"]}


# -- Table-3-shaped budget sweep ---------------------------------------------------------------
def run_budget_sweep(n_sessions: int) -> dict:
    """Budgets B in {unbounded, 8K, 6K, 4K, 0 (floor)} on full-size single sessions (32
    layers, 600 units, batch size 1, one session at a time): End and Peak resident
    positions (means over sessions, as the device reports them) and the path's GPU time per
    unit (append, every layer's attention and the evict of one unit; CUDA events), mean and
    p99.  SM clocks are sampled throughout."""
    import numpy as np
    import torch
    from synth import script as S
    from synth.driver import Driver
    rows = []
    clocks = Clocks(torch.cuda.current_device())
    clocks.start()
    for budget in (-1, 8192, 6144, 4096, 0):
        w = S.SINGLE_BF16.with_(name=f"single-bf16-32L-600u-B{budget}-W10", budget=budget,
                                n_sessions=n_sessions)
        ends, peaks, unit_ms = [], [], []
        for sid in range(n_sessions):
            drv = Driver(w, [S.session_script(w, sid)])
            spans = []
            for _ in range(len(drv.sched)):
                st = drv.prepare_step()
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                drv.run_step(st)
                e1.record()
                spans.append((e0, e1))
                del st
            torch.cuda.synchronize()
            unit_ms += [a.elapsed_time(b) for a, b in spans]
            info = drv.cache.export_state(sid)
            ends.append(info["resident"])
            peaks.append(info["peak_resident"])
            del drv
            torch.cuda.empty_cache()
        t = np.array(unit_ms)
        rows.append({"budget": "unbounded" if budget < 0 else budget,
                     "end_positions": float(np.mean(ends)), "peak_positions": float(np.mean(peaks)),
                     "end_per_session": ends, "peak_per_session": peaks,
                     "unit_ms_mean": float(t.mean()), "unit_ms_p99": float(np.percentile(t, 99)),
                     "units": int(t.size)})
    clk = clocks.stop()
    full = rows[0]["peak_positions"]
    for r in rows:
        r["peak_reduction_vs_unbounded"] = 1.0 - r["peak_positions"] / full
    return {"sweep": "Table-3-shaped budget sweep, synthetic single-session workload "
                     "(32 layers, 32/8 heads, D=128, bf16, W=10, 600 units, batch size 1)",
            "data": "synthetic (seeded SplitMix64 Irwin-Hall values, PCG64 session scripts)",
            "sessions_per_budget": n_sessions, "rows": rows, "clocks": clk}


# -- the stress workload at scale ------------------------------------------------------------
def run_stress(budget: int, window: int, n_sessions: int, steps: int, warmup: int) -> dict:
    """The stress workload (10-60 minute sessions, 5 % units without a segment, 2 % long
    segments of 10-30 tokens) at one (B, W) grid point with `n_sessions` concurrent
    sessions: the cache is brought (append + evict only) to the step where every session
    is at its budget, then `warmup` and `steps` timed steps of the whole path (append,
    every layer's attention, evict).  The scripts are cut after the last timed step, so
    the pool is sized for the positions fed until then."""
    import torch
    from synth import script as S
    from synth.driver import Driver
    w = S.stress256(budget, window).with_(n_sessions=n_sessions)
    scripts = S.workload_scripts(w)
    start = S.steady_state_step(w, scripts)
    keep = start + warmup + steps
    for sc in scripts:
        sc.n_transcript = sc.n_transcript[:keep]
        sc.n_text = sc.n_text[:keep]
    # Pool: each session's resident bound (budget or protected content, plus one unit) in
    # pages, plus ten pages for partly filled pages and the eviction's transient.
    from synth.driver import cache_sizing, resident_bound
    sizing = cache_sizing(w, scripts)
    sizing["n_pages"] = sum(resident_bound(w, sc)[0] // w.page_size + 10 for sc in scripts) + 16
    drv = Driver(w, scripts, sizing=sizing)
    drv.fast_forward(start)
    for _ in range(warmup):
        drv.run_step(drv.prepare_step())
    timed = [drv.prepare_step() for _ in range(steps)]
    torch.cuda.synchronize()
    clocks = Clocks(torch.cuda.current_device())
    clocks.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    launches = 0
    for st in timed:
        launches += drv.run_step(st)
    e1.record()
    torch.cuda.synchronize()
    clk = clocks.stop()
    ms = e0.elapsed_time(e1)
    audio_s = sum(len(st.pairs) for st in timed)
    resident = [drv.cache.export_state(sc.session)["resident"] for sc in scripts[:8]]
    return {"metric": METRIC, "value": audio_s / (ms / 1e3), "unit": UNIT, "steps": steps,
            "warmup": warmup, "ms_per_step": ms / steps, "higher_is_better": True,
            "dtype": w.dtype, "data": "synthetic (seeded SplitMix64 Irwin-Hall values, PCG64 "
                                       "session scripts)",
            "config": {"workload": w.name, "sessions": n_sessions, "budget": budget,
                       "window": window, "timed_steps": [start + warmup, keep],
                       "pool_pages": drv.sizing["n_pages"],
                       "resident_first_sessions": resident},
            "gpu_launches": launches, "clocks": clk}


# -- the oracle on the host cores -----------------------------------------------------------------
_BLAS_THREAD_VARS = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")


def _oracle_layers(session: int, start: int, layers: list) -> float:
    """One session's unit at step `start` of the 64-session workload through the oracle:
    the state before the unit is built untimed, then the unit's policy steps and every
    attention call of `layers` are timed.  Returns the timed seconds."""
    from oracle.cache import OracleCache, OracleConfig
    from synth import script as S
    from synth import values as V

    w = S.BATCH64_BF16
    sc = S.session_script(w, session)
    unit = start - sc.offset
    orc = OracleCache(OracleConfig(n_sessions=1, layers=w.layers, q_heads=w.q_heads,
                                   kv_heads=w.kv_heads, head_dim=w.head_dim,
                                   page_size=w.page_size, budget=w.budget, window=w.window,
                                   dtype=w.dtype, rope_base=w.rope_base, n_pages=1 << 20))
    for u in range(unit):           # state before the sampled unit (untimed)
        orc.append_chunk([0], [sc.unit_types(u)])
        orc.evict([0])

    def kv(s, layer, pos):
        return (V.layer_tensor(w.seed, V.TAG_K, session, layer, pos, w.kv_heads, w.head_dim,
                               w.dtype), V.layer_tensor(w.seed, V.TAG_V, session, layer, pos,
                                                        w.kv_heads, w.head_dim, w.dtype))

    t0 = time.perf_counter()
    chunks = [sc.prefill_types()] + [sc.decode_types(unit)[i:i + 1]
                                     for i in range(len(sc.decode_types(unit)))]
    for types in chunks:
        orc.append_chunk([0], [types])
        pos = orc.last_append[0][1]
        for layer in layers:
            q = V.layer_tensor(w.seed, V.TAG_Q, session, layer, pos, w.q_heads, w.head_dim,
                               w.dtype)
            orc.attend(layer, [q], kv)
    orc.evict([0])
    return time.perf_counter() - t0


def oracle_sample(layers_sampled: int = 1, session: int = 0, start: int | None = None,
                  workers: int = 1) -> dict:
    """Time the CPU oracle on one session's unit at the benchmark's steady state, for
    `layers_sampled` of its 32 layers (policy + every attention call of those layers),
    scaled to audio-s/s by the sampled fraction of one unit.

    workers = 1: one process with single-threaded BLAS.  workers = N: N processes
    (spawned; each single-threaded), layer i in process i % N, all replaying the unit's
    calls in parallel; the value is the sampled fraction over the wall time of the
    parallel part."""
    import multiprocessing as mp
    from synth import script as S
    w = S.BATCH64_BF16
    if start is None:
        start = S.steady_state_step(w, S.workload_scripts(w))
    unit = start - S.session_script(w, session).offset
    n_calls = 1 + len(S.session_script(w, session).decode_types(unit))
    saved = {k: os.environ.get(k) for k in _BLAS_THREAD_VARS}
    for k in _BLAS_THREAD_VARS:
        os.environ[k] = "1"
    try:
        ctx = mp.get_context("spawn")
        with ctx.Pool(workers) as pool:
            pool.apply(time.perf_counter)        # workers started before the clock
            parts = [list(range(i, layers_sampled, workers)) for i in range(workers)]
            t0 = time.perf_counter()
            pool.starmap(_oracle_layers, [(session, start, p) for p in parts if p])
            dt = time.perf_counter() - t0
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    frac = layers_sampled / w.layers
    return {"value": frac / dt, "unit": UNIT, "cores": workers, "kind": "oracle",
            "seconds": dt,
            "sample": f"session {session}, unit {unit} (step {start}) of {w.name}: eviction rule "
                      f"+ {n_calls} attention calls x {layers_sampled}/{w.layers} layers in "
                      f"float64, {workers} single-threaded process(es); value = sampled "
                      f"fraction of one audio-second / wall time"}


def cpu_baseline() -> dict:
    """The oracle on all host cores (the reported figure) and on one core."""
    cores = len(os.sched_getaffinity(0))
    allc = oracle_sample(layers_sampled=2 * cores, workers=cores)
    one = oracle_sample(layers_sampled=6, workers=1)
    allc["single_thread"] = {"value": one["value"], "cores": 1, "seconds": one["seconds"],
                             "sample": one["sample"]}
    return allc


def run_reference(args, rank: int, world: int):
    """The oracle timed as the reference arm (host cores), same metric and unit."""
    if rank != 0:
        return None
    from synth import script as S
    w = S.BATCH64_BF16
    start = S.steady_state_step(w, S.workload_scripts(w))
    # Each step: one session-unit of the steady state, 1 of its 32 layers (sessions taken
    # in turn); W untimed samples first.
    cores = len(os.sched_getaffinity(0))
    for i in range(args.warmup):
        oracle_sample(layers_sampled=cores, session=(args.steps + i) % w.n_sessions,
                      start=start, workers=cores)
    samples = [oracle_sample(layers_sampled=cores, session=i % w.n_sessions, start=start,
                             workers=cores) for i in range(args.steps)]
    total_audio = sum(s["value"] * s["seconds"] for s in samples)
    total_t = sum(s["seconds"] for s in samples)
    v = total_audio / total_t
    sample = ("%d of 32 layers of one session-unit per step (sessions in turn, step %d), one "
              "layer per single-threaded process on %d host cores" % (cores, start, cores))
    return {
        "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * total_t / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded SplitMix64 Irwin-Hall values, PCG64 session scripts)",
        "impl": "reference",
        "config": dict(workload_config(w, start, args.steps, world, False), sample=sample),
        "cpu_baseline": {"value": v, "unit": UNIT, "kind": "oracle",
                         "cores": samples[0]["cores"], "sample": sample},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--start", type=int, default=None, help="first timed step of the schedule")
    ap.add_argument("--e2e-steps", type=int, default=None)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--compare-unbounded", action="store_true",
                    help="print the B=4096 vs B=infinity single-session comparison and exit")
    ap.add_argument("--per-layer-append", action="store_true",
                    help="the model's order: appends without K/V, each layer's K/V written "
                         "just before its attention")
    ap.add_argument("--budget-sweep", type=int, default=0, metavar="SESSIONS",
                    help="print the Table-3-shaped budget sweep over SESSIONS sessions and exit")
    ap.add_argument("--stress", default=None, metavar="B,W[,N]",
                    help="print one JSON line for the stress workload at budget B, window W "
                         "with N concurrent sessions (default 256) and exit")
    ap.add_argument("--sessions", type=int, default=None,
                    help="reduced case for profiler captures (default: the full 64)")
    ap.add_argument("--layers", type=int, default=None,
                    help="reduced case for profiler captures (default: the full 32)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)

    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local_rank = int(os.environ.get("LOCAL_RANK", 0))
    if world > 1 and args.impl == "ours":
        import torch
        torch.distributed.init_process_group(
            backend="nccl" if torch.cuda.is_available() else "gloo")

    if args.impl == "reference":
        out = run_reference(args, rank, world)
        if out is not None:
            print(json.dumps(out))
        return

    from __graft_entry__ import build
    build()
    if args.compare_unbounded:
        if rank == 0:
            print(json.dumps(run_unbounded_comparison()))
        return
    if args.budget_sweep:
        if rank == 0:
            print(json.dumps(run_budget_sweep(args.budget_sweep)))
        return
    if args.stress:
        if rank == 0:
            f = [int(x) for x in args.stress.split(",")]
            print(json.dumps(run_stress(f[0], f[1], f[2] if len(f) > 2 else 256, args.steps,
                                        args.warmup)))
        return
    out = run_ours(args, rank, world, local_rank)
    if rank == 0:
        if world == 1 and not args.no_cpu_baseline:
            out["cpu_baseline"] = cpu_baseline()
        print(json.dumps(out))
    if world > 1:
        import torch
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
