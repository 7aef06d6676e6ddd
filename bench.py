"""Timing of the STEPQuant decode step on the 1024-slot serving pool.

One step = one decode token through all 16 recurrent layers for the 1024 active
slots (16 launches of the fused kernel, one per layer), i.e. 524,288 head-state
updates. Prints one JSON line (see the keys below). `--impl reference` times
the CPU oracle on a bounded sample of the same workload instead.

Multi-GPU: every (slot, layer, head) update is independent and the path has no
exchange step, so N ranks run N independent replicas of the workload (weak
scaling, no collective on the data path); the value sums all ranks' updates
over the slowest rank's time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "head-state decode updates/sec and achieved HBM GB/s (fraction of peak) at 1 GB300"
UNIT = "head-updates/s"
WORKLOAD = "pool"


def _peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return {}


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 100 ms by one
    nvidia-smi process that runs across every timed region."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        rows = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=10)
            except Exception:
                self.proc.kill()
                out, _ = self.proc.communicate()
            rows = [[x.strip() for x in line.split(",")] for line in out.splitlines() if line.strip()]
        sm = [float(r[0]) for r in rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in rows if len(r) > 1 and r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in rows for k in range(4)
                          if len(r) > 3 + k and r[3 + k].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


def _cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the machine type)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.machine()


def _recorded_traffic(units_per_launch: int):
    """DRAM bytes per launch of the fused kernel from the committed ncu record,
    or None once the kernel's sources differ from the ones that were measured."""
    import hashlib
    try:
        rec = json.load(open(os.path.join(ROOT, "profiles", "decode_heads_pool.traffic.json")))
        h = hashlib.sha256()
        for f in rec["source_files"]:
            h.update(open(os.path.join(ROOT, f), "rb").read())
        if h.hexdigest()[:16] != rec["source_sha256_16"]:
            return None
        return rec["dram_bytes_per_head_update"] * units_per_launch
    except Exception:
        return None


def reduce_over_ranks(total_ms: float, units: float, world: int, device=None):
    """Max of the timed region over ranks and the whole-job rate: every rank runs
    its own replica, so all ranks' units count over the slowest rank's time."""
    if world > 1:
        import torch
        import torch.distributed as dist
        t = torch.tensor([float(total_ms)], dtype=torch.float64,
                         device=device if device is not None else "cpu")
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
    return total_ms, world * units / (total_ms / 1e3)


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def cpu_baseline(wl, units: int, min_seconds: float = 10.0):
    """The oracle as it stands, on a bounded sample of the workload (all host cores):
    decode steps of one layer for units / 32 slots, repeated until `min_seconds`."""
    import oracle as O
    from paper_2609_38169_gb300 import workloads as W
    wl1 = wl.replace(layers=1)
    st = O.calibrate(wl1, seqs=2, steps=16)
    oplan = O.plan_from_stats(wl1, st)
    mp = W.model_params(wl)
    B = max(1, units // wl.hv)
    slots = np.arange(B, dtype=np.int32)
    S = W.random_states(wl, B * wl.hv).reshape(B, wl.hv, 128, 128)
    pool = np.zeros(B * oplan.slot_stride, np.uint8)
    O.pool_encode(oplan, pool, 0, slots, S)
    del S
    done, elapsed, step = 0, 0.0, 0
    while elapsed < min_seconds or step == 0:
        inp = W.step_inputs(wl, mp, W.STREAM_DECODE, step, 0, batch=B)
        t0 = time.perf_counter()
        O.pool_step(oplan, pool, 0, slots, inp)
        elapsed += time.perf_counter() - t0
        done += B * wl.hv
        step += 1
    return {"value": done / elapsed, "unit": UNIT, "cores": O.num_threads(), "kind": "oracle",
            "cpu_model": _cpu_model(),
            "sample": f"{step} decode steps of one layer for {B} slots x {wl.hv} heads "
                      f"({done} head updates) of the {wl.name} workload, {elapsed:.1f} s"}


def secondary_channel(args, dev, peak, _unused=None):
    """The channel-gate decode workload (one layer of 32 heads with per-key-channel
    gates, 256 slots, STEPQuant at 4 bits: row units) beside the FP32-state and
    INT8 rowwise kernels on the same inputs. Its pool is smaller than L2, so a
    256 MiB buffer is written between timed launches and only the launches are
    timed (CUDA events around each)."""
    import torch
    import paper_2609_38169_gb300 as P
    from paper_2609_38169_gb300 import workloads as W
    wl = W.WORKLOADS["channel"]
    cfg = P.Config.from_workload(wl)
    Hv, Hk, B = wl.hv, wl.hk, wl.batch
    st = P.calibrate(cfg, wl, device=dev, steps=min(args.calib_steps, wl.calib_steps), device_inputs=True)
    plan = P.stepq_fit_scales(cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
    mp_dev = W.model_params_torch(W.model_params(wl), dev)
    fp32_pool = torch.zeros((wl.pool_slots, 1, Hv, 128, 128), dtype=torch.float32, device=dev)
    all_slots = torch.arange(wl.pool_slots, dtype=torch.int32, device=dev)
    y = torch.empty((B, Hv, 128), dtype=torch.float32, device=dev)
    for t in range(wl.warmup_steps):
        q, k, v, beta, gate = W.torch_step_inputs(wl, mp_dev, t, 0, dev, W.STREAM_WARMUP, batch=wl.pool_slots)
        P.stepq_fp32_decode_step(cfg, 0, fp32_pool, all_slots, q, k, v, beta, gate, y)
    pool = P.alloc_pool(plan, wl.pool_slots, dev)
    P.stepq_quantize_pool(plan, 0, fp32_pool, all_slots, pool)
    i8_stride = P.stepq_intb_slot_bytes(cfg, 8)
    i8_pool = torch.zeros(wl.pool_slots * i8_stride, dtype=torch.uint8, device=dev)
    P.stepq_intb_quantize_pool(cfg, 8, 0, fp32_pool, all_slots, i8_pool)
    slots = torch.from_numpy(W.slot_permutation(wl)).to(dev)
    inputs = [W.torch_step_inputs(wl, mp_dev, 1000 + s, 0, dev) for s in range(2)]
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def timed(call, steps, warmup):
        for s in range(warmup):
            call(*inputs[s % 2])
        torch.cuda.synchronize(dev)
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(steps)]
        for s in range(steps):
            flush.fill_(s & 0xFF)                         # L2 holds none of the pool
            evs[s][0].record(stream)
            call(*inputs[s % 2])
            evs[s][1].record(stream)
        torch.cuda.synchronize(dev)
        return [a.elapsed_time(b) for a, b in evs]

    steps = max(args.steps, 10)
    ms = timed(lambda q, k, v, beta, gate: P.stepq_decode_step(plan, 0, pool, slots, q, k, v, beta, gate, y,
                                                                pool_slots=wl.pool_slots), steps, args.warmup)
    fp_ms = timed(lambda q, k, v, beta, gate: P.stepq_fp32_decode_step(cfg, 0, fp32_pool, slots, q, k, v, beta,
                                                                        gate, y, pool_slots=wl.pool_slots),
                  steps, args.warmup)
    i8_ms = timed(lambda q, k, v, beta, gate: P.stepq_intb_decode_step(cfg, 8, 0, i8_pool, slots, q, k, v, beta,
                                                                        gate, y, pool_slots=wl.pool_slots),
                  steps, args.warmup)
    assert P.stepq_device_error() == 0
    units = B * Hv
    io_b = B * (Hk * 2 * 512 + Hv * (512 + 4 + 512 + 512))
    page_b = int(B * 2 * plan.head_bytes.astype(np.int64).sum())
    avg = statistics.mean(ms) / 1e3
    achieved = (page_b + io_b) / avg / 1e9
    fp_b = units * 2 * 65536 + io_b
    i8_b = units * 2 * (i8_stride // Hv) + io_b
    out = {"workload": "channel-wise gate decode: 1 layer x 32 heads, d=128, 256 slots (random permutation), "
                       "per-key-channel gates, STEPQuant @4 (row units); L2 flushed between launches",
           "metric": "head-state decode updates/sec (one layer launch)", "unit": UNIT,
           "value": units / avg, "ms_per_launch": avg * 1e3,
           "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                        "frac": achieved / peak, "traffic": None, "bytes_per_launch": page_b + io_b,
                        "avg_launch_us": avg * 1e6},
           "baselines": {
               "fp32_state": {"value": units / (statistics.mean(fp_ms) / 1e3), "ms_per_launch": statistics.mean(fp_ms),
                              "achieved_gbs": fp_b / (statistics.mean(fp_ms) / 1e3) / 1e9},
               "int8_rowwise": {"value": units / (statistics.mean(i8_ms) / 1e3), "ms_per_launch": statistics.mean(i8_ms),
                                "achieved_gbs": i8_b / (statistics.mean(i8_ms) / 1e3) / 1e9}},
           "cpu_baseline": None}
    if not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(wl, 512, min_seconds=5.0)
    return out


def run_reference(args):
    """The CPU oracle timed as the reference arm (rank 0 only)."""
    world, rank, _ = dist_setup()
    if rank != 0:
        return
    from paper_2609_38169_gb300 import workloads as W
    wl = W.WORKLOADS[WORKLOAD]
    per_step_units = args.ref_units
    vals = []
    for _ in range(args.warmup):
        cpu_baseline(wl, per_step_units, min_seconds=0.0)
    for _ in range(args.steps):
        vals.append(cpu_baseline(wl, per_step_units, min_seconds=0.0))
    v = statistics.median(x["value"] for x in vals)
    ms = 1e3 * per_step_units / v
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": "serving state pool: 16 layers x 32 heads, 1024 slots, d=128, "
                                   "nominal 6-bit STEPQuant (oracle on a bounded sample)",
                       "sample_units_per_step": per_step_units},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": vals[-1]["cores"], "kind": "oracle",
                             "sample": vals[-1]["sample"]},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="stepq", choices=["stepq", "reference"])
    ap.add_argument("--no-baselines", action="store_true")
    ap.add_argument("--no-secondary", action="store_true", help="skip the channel-gate row-unit line")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-units", type=int, default=4096)
    ap.add_argument("--ref-units", type=int, default=1024)
    ap.add_argument("--calib-steps", type=int, default=256)
    ap.add_argument("--slots", type=int, default=None, help="smaller pool (profiling cases only)")
    ap.add_argument("--layers", type=int, default=None, help="fewer layers (profiling cases only)")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)

    import torch
    import paper_2609_38169_gb300 as P
    from paper_2609_38169_gb300 import workloads as W

    world, rank, local = dist_setup()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    wl = W.WORKLOADS[WORKLOAD]
    if args.slots or args.layers:
        wl = wl.replace(batch=args.slots or wl.batch, pool_slots=args.slots or wl.pool_slots,
                        layers=args.layers or wl.layers)
    cfg = P.Config.from_workload(wl)
    L, Hv, Hk, B = wl.layers, wl.hv, wl.hk, wl.batch

    # ---- offline: calibration and plan (not timed) ----
    st = P.calibrate(cfg, wl, device=dev, steps=args.calib_steps, device_inputs=True)
    plan = P.stepq_fit_scales(cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
    mp_dev = W.model_params_torch(W.model_params(wl), dev)

    # ---- initial states: 32 FP32 warm-up steps from zero, then pack ----
    fp32_pool = torch.zeros((wl.pool_slots, L, Hv, 128, 128), dtype=torch.float32, device=dev)
    all_slots = torch.arange(wl.pool_slots, dtype=torch.int32, device=dev)
    y_tmp = torch.empty((wl.pool_slots, Hv, 128), dtype=torch.float32, device=dev)
    for t in range(wl.warmup_steps):
        for layer in range(L):
            q, k, v, beta, gate = W.torch_step_inputs(wl, mp_dev, t, layer, dev, W.STREAM_WARMUP,
                                                      batch=wl.pool_slots)
            P.stepq_fp32_decode_step(cfg, layer, fp32_pool, all_slots, q, k, v, beta, gate, y_tmp)
    pool = P.alloc_pool(plan, wl.pool_slots, dev)
    P.stepq_quantize_pool(plan, -1, fp32_pool, all_slots, pool)
    int8_stride = P.stepq_intb_slot_bytes(cfg, 8)
    int8_pool = None
    if not args.no_baselines:
        int8_pool = torch.zeros(wl.pool_slots * int8_stride, dtype=torch.uint8, device=dev)
        P.stepq_intb_quantize_pool(cfg, 8, -1, fp32_pool, all_slots, int8_pool)
    else:
        del fp32_pool
        fp32_pool = None
    torch.cuda.synchronize()
    assert P.stepq_device_error() == 0

    slots = torch.from_numpy(W.slot_permutation(wl)).to(dev)
    n_inputs = 2                       # distinct token steps of inputs, cycled
    inputs = [[W.torch_step_inputs(wl, mp_dev, 1000 + s, layer, dev) for layer in range(L)]
              for s in range(n_inputs)]
    y = torch.empty((L, B, Hv, 128), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step_stepq(s, ev=None):
        for layer in range(L):
            q, k, v, beta, gate = inputs[s % n_inputs][layer]
            if ev is not None:
                ev[layer][0].record(stream)
            P.stepq_decode_step(plan, layer, pool, slots, q, k, v, beta, gate, y[layer],
                                pool_slots=wl.pool_slots)
            if ev is not None:
                ev[layer][1].record(stream)

    def step_fp32(s):
        for layer in range(L):
            q, k, v, beta, gate = inputs[s % n_inputs][layer]
            P.stepq_fp32_decode_step(cfg, layer, fp32_pool, slots, q, k, v, beta, gate, y[layer],
                                     pool_slots=wl.pool_slots)

    def step_int8(s):
        for layer in range(L):
            q, k, v, beta, gate = inputs[s % n_inputs][layer]
            P.stepq_intb_decode_step(cfg, 8, layer, int8_pool, slots, q, k, v, beta, gate, y[layer],
                                     pool_slots=wl.pool_slots)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize(dev)

    wall_s = {}                                        # host wall time of each timed region

    def timed(fn, steps, warmup, per_launch=False, name="timed"):
        for s in range(warmup):
            fn(s)
        evs = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                for _ in range(L)] for _ in range(steps)] if per_launch else None
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.nvtx.range_push(name)
        e0.record(stream)
        w0 = time.perf_counter()
        for s in range(steps):
            if per_launch:
                fn(s, evs[s])
            else:
                fn(s)
        e1.record(stream)
        torch.cuda.nvtx.range_pop()
        barrier()
        wall_s[name] = time.perf_counter() - w0
        total_ms = e0.elapsed_time(e1)
        launch_ms = None
        if per_launch:
            launch_ms = [a.elapsed_time(b) for row in evs for (a, b) in row]
        return total_ms, launch_ms

    clocks = ClockSampler(dev.index if dev.index is not None else 0)
    clocks.start()
    total_ms, launch_ms = timed(step_stepq, args.steps, args.warmup, per_launch=True, name="stepq_decode")
    assert P.stepq_device_error() == 0
    units_per_step = L * B * Hv
    total_ms, value = reduce_over_ranks(total_ms, units_per_step * args.steps, world, dev)

    # algorithmic bytes per launch: each head page read and written once, plus
    # q, k (per key head), v, beta, gate read and y written
    head_bytes = plan.head_bytes.reshape(L, Hv).astype(np.int64)
    gate_b = 4 * (128 if cfg.unit_rows else 1)
    io_b = B * (Hk * 2 * 512 + Hv * (512 + 4 + gate_b + 512))
    layer_bytes = [int(B * 2 * head_bytes[l].sum() + io_b) for l in range(L)]
    avg_launch_s = statistics.mean(launch_ms) / 1e3
    achieved = statistics.mean(layer_bytes) / avg_launch_s / 1e9
    peaks = _peaks()
    peak = peaks.get("hbm_gbs", 6800.0)
    traffic = _recorded_traffic(B * Hv) if (L, B, Hv) == (16, 1024, 32) else None
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": traffic,
                "peak_source": "measured" if "hbm_gbs" in peaks else "fallback",
                "bytes_per_launch": statistics.mean(layer_bytes),
                "avg_launch_us": avg_launch_s * 1e6,
                "median_launch_us": statistics.median(launch_ms) * 1e3}

    # ---- end to end through the public API with host buffers ----
    # Every step copies each layer's inputs from pinned host memory and reads
    # every layer's y back. The copies run on their own streams, up to two
    # layers ahead of / one behind the kernel that uses them (three device
    # input buffers, ordered by events), so they overlap the decode kernels;
    # the step ends when the last y has reached the host.
    # a layer's five inputs travel as one packed buffer (one copy per layer);
    # the library gets a view of each
    shapes = [x.shape for x in inputs[0][0]]
    sizes = [x.numel() for x in inputs[0][0]]
    total = sum(sizes)

    def views(flat):
        out, o = [], 0
        for shp, n in zip(shapes, sizes):
            out.append(flat[o:o + n].view(shp))
            o += n
        return out

    h_in = []
    for layer in range(L):
        flat = torch.empty(total, dtype=torch.float32).pin_memory()
        for dst, src in zip(views(flat), inputs[0][layer]):
            dst.copy_(src)
        h_in.append(flat)
    n_buf = 3
    d_flat = [torch.empty(total, dtype=torch.float32, device=dev) for _ in range(n_buf)]
    d_in = [views(f) for f in d_flat]
    h_y = torch.empty((L, B, Hv, 128), dtype=torch.float32).pin_memory()
    h2d = sum(x.numel() * x.element_size() for x in h_in)
    d2h = h_y.numel() * 4
    h2d_stream, d2h_stream = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    buf_free = [torch.cuda.Event() for _ in range(n_buf)]
    copied = [torch.cuda.Event() for _ in range(n_buf)]
    y_done = [torch.cuda.Event() for _ in range(L)]
    y_read = [torch.cuda.Event() for _ in range(L)]
    lookahead = 2
    step_done = [torch.cuda.Event() for _ in range(lookahead + 1)]
    for e in buf_free + y_read:
        e.record(stream)

    def step_e2e(s):
        # At most `lookahead` steps in flight, as a serving loop keeps them. An
        # unbounded loop fills the launch queue, and the host then blocks on the
        # decode stream while the next layers' input copies, on their own
        # stream, are not yet issued.
        if s >= lookahead:
            step_done[(s - lookahead) % (lookahead + 1)].synchronize()
        for layer in range(L):
            nb = (s * L + layer) % n_buf
            h2d_stream.wait_event(buf_free[nb])         # the kernel that last read this buffer
            with torch.cuda.stream(h2d_stream):
                d_flat[nb].copy_(h_in[layer], non_blocking=True)
                copied[nb].record(h2d_stream)
            stream.wait_event(copied[nb])
            stream.wait_event(y_read[layer])            # last step's y of this layer is on the host
            q, k, v, beta, gate = d_in[nb]
            P.stepq_decode_step(plan, layer, pool, slots, q, k, v, beta, gate, y[layer],
                                pool_slots=wl.pool_slots, stream=stream)
            buf_free[nb].record(stream)
            y_done[layer].record(stream)
            d2h_stream.wait_event(y_done[layer])
            with torch.cuda.stream(d2h_stream):
                h_y[layer].copy_(y[layer], non_blocking=True)
                y_read[layer].record(d2h_stream)
        stream.wait_event(y_read[L - 1])                # the step ends with y on the host
        step_done[s % (lookahead + 1)].record(stream)

    e2e_steps = max(3, args.steps // 2)
    # three end-to-end regions; the median is reported (host-side copy scheduling varies)
    e2e_values = []
    for rep in range(3):
        e2e_ms, _ = timed(step_e2e, e2e_steps, 2, name=f"stepq_e2e{rep}")
        e2e_values.append(reduce_over_ranks(e2e_ms, units_per_step * e2e_steps, world, dev)[1])
    e2e = {"value": statistics.median(e2e_values), "unit": UNIT, "h2d_bytes_per_step": h2d,
           "d2h_bytes_per_step": d2h, "regions": e2e_values}

    baselines = {}
    if not args.no_baselines:
        nb = max(3, args.steps // 2)
        fp_ms, _ = timed(step_fp32, nb, 2, name="fp32_decode")
        i8_ms, _ = timed(step_int8, nb, 2, name="int8_decode")
        fp_bytes = B * Hv * (2 * 65536) + io_b
        i8_bytes = B * Hv * 2 * (256 + 16384) + io_b
        baselines = {
            "fp32_state": {"value": units_per_step * nb / (fp_ms / 1e3), "unit": UNIT,
                           "ms_per_step": fp_ms / nb,
                           "achieved_gbs": L * fp_bytes * nb / (fp_ms / 1e3) / 1e9},
            "int8_rowwise": {"value": units_per_step * nb / (i8_ms / 1e3), "unit": UNIT,
                             "ms_per_step": i8_ms / nb,
                             "achieved_gbs": L * i8_bytes * nb / (i8_ms / 1e3) / 1e9},
        }
    clk = clocks.stop()
    secondary = None
    if not args.no_secondary and world == 1:
        secondary = secondary_channel(args, dev, peak, None)

    if rank == 0:
        cpu = None
        if not args.no_cpu_baseline and world == 1:
            cpu = cpu_baseline(wl, args.cpu_units)
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": f"serving state pool: {L} Delta-rule layers x {Hv} heads, d_k=d_v=128, "
                                   f"{B} request slots (random permutation), nominal 6-bit STEPQuant, "
                                   f"one step = one token through all {L} layers",
                       "layers": L, "heads": Hv, "slots": B, "pool_bytes": plan.slot_stride * wl.pool_slots,
                       "slot_stride": plan.slot_stride, "l2": f"inputs larger than L2 (pool {plan.slot_stride * wl.pool_slots / 1e9:.2f} GB)",
                       "parallelism": f"replicas x{world}"},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": L * args.steps, "clocks": clk, "baselines": baselines,
            "secondary": secondary,
            "wall_s": {k: round(v, 4) for k, v in wall_s.items()},
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
