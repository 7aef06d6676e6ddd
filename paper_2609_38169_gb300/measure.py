"""Measurements of the kernels beside the headline decode step (which bench.py
times): the row-unit decode step against the FP32-state and INT-b comparison
kernels on one layer of a channel-gate pool, and the chunked FP32 prefill.
Each subcommand prints one JSON line; inputs are synthetic (the workload
generators), resident on the device, and timed with CUDA events after warm-up.

    python -m paper_2609_38169_gb300.measure rows [--slots 1024] [--bits 6]
    python -m paper_2609_38169_gb300.measure prefill [--slots 128] [--tokens 512]
    python -m paper_2609_38169_gb300.measure split [--slots 1024] [--layers 16]
    python -m paper_2609_38169_gb300.measure calib [--workload pool]
"""
from __future__ import annotations

import argparse
import json

from . import api as A, workloads as W

D = 128
FP32_FMA_PEAK_FLOPS = 128 * 2 * 152 * 2.07e9     # FMA lanes/clk/SM x 2 x SMs x max SM clock


def _timeit(fn, n=20, warmup=3):
    import torch
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(n):
        fn()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / n * 1e-3          # seconds per call


def rows(slots=1024, bits=6):
    """One layer of the drift workload's shape (32 heads, channel gates) over
    `slots` slots in a random permutation: STEPQuant row units against the
    FP32-state and INT8 / INT6 rowwise kernels on identical inputs."""
    import torch
    dev = torch.device("cuda")
    wl = W.WORKLOADS["drift"].replace(layers=1, batch=slots, pool_slots=slots, nominal_bits=bits,
                                      candidates=(4, 6, 8) if bits == 6 else (2, 4, 6, 8))
    cfg = A.Config.from_workload(wl)
    st = A.calibrate(cfg, wl, dev, seqs=4, steps=64, device_inputs=True)
    plan = A.stepq_fit_scales(cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    S = torch.randn((slots, 1, wl.hv, D, D), generator=g, device=dev)
    S *= torch.exp(torch.randn((slots, 1, wl.hv, D, 1), generator=g, device=dev))
    all_slots = torch.arange(slots, dtype=torch.int32, device=dev)
    perm = torch.from_numpy(W.slot_permutation(wl)).to(dev)
    pool = A.alloc_pool(plan, slots, dev)
    A.stepq_quantize_pool(plan, -1, S, all_slots, pool)
    q, k, v, beta, gate = W.torch_step_inputs(wl, W.model_params_torch(W.model_params(wl), dev), 0, 0, dev)
    y = torch.empty((slots, wl.hv, D), device=dev)
    units = slots * wl.hv
    vec = 4 * 512 + 512 + 4                                    # q k v gate y beta per head update
    out = {"metric": "row-unit decode step, one layer", "unit": "head-updates/s",
           "workload": f"{slots} slots x {wl.hv} heads, channel gates, STEPQuant @{bits}",
           "kernels": {}}
    t = _timeit(lambda: A.stepq_decode_step(plan, 0, pool, perm, q, k, v, beta, gate, y))
    page = plan.slot_stride / wl.hv
    out["kernels"]["stepq_rows"] = {"us_per_launch": t * 1e6, "value": units / t,
                                    "algorithmic_gbs": units * (2 * page + vec) / t / 1e9,
                                    "bits_per_value": 8 * page / (D * D)}
    ref = S.clone()
    t = _timeit(lambda: A.stepq_fp32_decode_step(cfg, 0, ref, perm, q, k, v, beta, gate, y))
    out["kernels"]["fp32_state"] = {"us_per_launch": t * 1e6, "value": units / t,
                                    "algorithmic_gbs": units * (2 * 4 * D * D + vec) / t / 1e9}
    for b in (8, 6):
        sb = A.stepq_intb_slot_bytes(cfg, b)
        pi = torch.zeros(slots * sb, dtype=torch.uint8, device=dev)
        A.stepq_intb_quantize_pool(cfg, b, -1, S, all_slots, pi)
        t = _timeit(lambda: A.stepq_intb_decode_step(cfg, b, 0, pi, perm, q, k, v, beta, gate, y))
        out["kernels"][f"int{b}_rowwise"] = {"us_per_launch": t * 1e6, "value": units / t,
                                             "algorithmic_gbs": units * (2 * sb / wl.hv + vec) / t / 1e9}
        del pi
    assert A.stepq_device_error() == 0
    return out


def prefill(slots=128, tokens=512, name="gqa"):
    """Chunked FP32 prefill of `tokens` tokens for `slots` slots of one layer."""
    import torch
    dev = torch.device("cuda")
    wl = W.WORKLOADS[name].replace(batch=slots, pool_slots=slots)
    cfg = A.Config.from_workload(wl)
    mp = W.model_params_torch(W.model_params(wl), dev)
    steps = [W.torch_step_inputs(wl, mp, t, 0, dev) for t in range(tokens)]
    q, k, v, beta, gate = [torch.stack([s[i] for s in steps], dim=1).contiguous() for i in range(5)]
    del steps
    states = torch.zeros((slots, wl.hv, D, D), device=dev)
    y = torch.empty((slots, tokens, wl.hv, D), device=dev)
    t = _timeit(lambda: A.stepq_prefill_fp32(cfg, states, q, k, v, beta, gate, y), n=5, warmup=2)
    head_tokens = slots * tokens * wl.hv
    C = 32
    # tensor-core work issued per chunk of one head (3 TF32 MMAs per split product):
    # P0 128 x 32 x 128, P1 128 x 64 x 128, P2 128 x 128 x 32, P3 128 x 32 x 32
    mma_flops = 3 * 2 * 128 * (32 * 128 + 64 * 128 + 128 * 32 + 32 * 32) / C
    # the fp32 work of the chunkwise form per head-token: K~S, Q~S and the state
    # update (3 x 128 x 128 FMAs), A and Q~K^T (2 x C x 128), the solve and Bm W (1.5 x C x 128)
    fma = 3 * D * D + 2 * C * D + 1.5 * C * D
    peak, src = tf32_peak()
    assert A.stepq_device_error() == 0
    return {"metric": "chunked FP32 prefill", "unit": "head-tokens/s", "value": head_tokens / t,
            "tokens_per_s": slots * tokens / t, "ms_per_call": t * 1e3,
            "workload": f"{name}: {slots} slots x {wl.hv} heads x {tokens} tokens",
            "roofline": {"bound": "tensor", "achieved": mma_flops * head_tokens / t / 1e12,
                         "peak": peak / 1e12, "unit": "TFLOP/s",
                         "frac": mma_flops * head_tokens / t / peak, "peak_source": src},
            "fp32_equivalent_tflops": 2 * fma * head_tokens / t / 1e12}


def tf32_peak():
    """Dense TF32 tensor peak: the measured bf16 GEMM rate times the nominal
    TF32 / BF16 ratio (1.1 / 2.25 PFLOP/s), or the fallback bf16 figure."""
    import os
    path = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            bf16 = float(json.load(f)["bf16_tflops"]) * 1e12
        src = "measured bf16 x nominal tf32/bf16"
    except (OSError, KeyError, ValueError):
        bf16, src = 1.9e15, "fallback bf16 x nominal tf32/bf16"
    return bf16 * 1.1 / 2.25, src


def split(slots=1024, layers=16):
    """The serving pool's decode step fused and split (Sec. 4.4, App. F.1).

    Per-launch times of one layer for the fused kernel, the readout and the
    writeback; then one token through all layers three ways: fused launches on
    one stream; readout and writeback on one stream; readout on the main
    stream with each writeback on a side stream ordered by an event (the
    paper's arrangement). For the side-stream form the time until the last
    layer's y is ready on the main stream is reported beside the total."""
    import torch
    dev = torch.device("cuda")
    wl = W.WORKLOADS["pool"].replace(layers=layers, batch=slots, pool_slots=slots)
    cfg = A.Config.from_workload(wl)
    st = A.calibrate(cfg, wl, dev, seqs=4, steps=64, device_inputs=True)
    plan = A.stepq_fit_scales(cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
    pool = A.alloc_pool(plan, slots, dev)
    all_slots = torch.arange(slots, dtype=torch.int32, device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(11)
    S = torch.empty((slots, 1, wl.hv, D, D), device=dev)
    for layer in range(layers):
        S.normal_(generator=g)
        A.stepq_quantize_pool(plan, layer, S[:, 0], all_slots, pool)
    del S
    perm = torch.from_numpy(W.slot_permutation(wl)).to(dev)
    mp = W.model_params_torch(W.model_params(wl), dev)
    inp = [W.torch_step_inputs(wl, mp, 0, layer, dev) for layer in range(layers)]
    y = torch.empty((layers, slots, wl.hv, D), device=dev)
    delta = torch.empty_like(y)
    units = slots * wl.hv
    out = {"metric": "side-stream split of the decode step", "unit": "us",
           "workload": f"pool: {layers} layers x {slots} slots x {wl.hv} heads, STEPQuant @6",
           "per_launch_us": {}}
    q, k, v, beta, gate = inp[0]
    out["per_launch_us"]["fused"] = 1e6 * _timeit(
        lambda: A.stepq_decode_step(plan, 0, pool, perm, q, k, v, beta, gate, y[0]))
    out["per_launch_us"]["readout"] = 1e6 * _timeit(
        lambda: A.stepq_decode_readout(plan, 0, pool, perm, q, k, v, beta, gate, y[0], delta[0]))
    out["per_launch_us"]["writeback"] = 1e6 * _timeit(
        lambda: A.stepq_decode_writeback(plan, 0, pool, perm, k, beta, gate, delta[0]))

    main, side = torch.cuda.current_stream(), torch.cuda.Stream()

    def fused():
        for layer in range(layers):
            q, k, v, beta, gate = inp[layer]
            A.stepq_decode_step(plan, layer, pool, perm, q, k, v, beta, gate, y[layer])

    def serial():
        for layer in range(layers):
            q, k, v, beta, gate = inp[layer]
            A.stepq_decode_readout(plan, layer, pool, perm, q, k, v, beta, gate, y[layer], delta[layer])
            A.stepq_decode_writeback(plan, layer, pool, perm, k, beta, gate, delta[layer])

    def two_streams(marks):
        marks[0].record(main)
        for layer in range(layers):
            q, k, v, beta, gate = inp[layer]
            A.stepq_decode_readout(plan, layer, pool, perm, q, k, v, beta, gate, y[layer],
                                   delta[layer], stream=main)
            ready = torch.cuda.Event()
            ready.record(main)
            side.wait_event(ready)
            A.stepq_decode_writeback(plan, layer, pool, perm, k, beta, gate, delta[layer], stream=side)
        marks[1].record(main)                        # the last y is ready
        done = torch.cuda.Event()
        done.record(side)
        main.wait_event(done)                        # writeback before the next token
        marks[2].record(main)

    n = 10
    out["token_ms"] = {"fused": 1e3 * _timeit(fused, n=n), "split_one_stream": 1e3 * _timeit(serial, n=n)}
    for _ in range(3):
        two_streams([torch.cuda.Event(enable_timing=True) for _ in range(3)])
    torch.cuda.synchronize()
    to_y, total = [], []
    for _ in range(n):
        marks = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        two_streams(marks)
        torch.cuda.synchronize()
        to_y.append(marks[0].elapsed_time(marks[1]))
        total.append(marks[0].elapsed_time(marks[2]))
    out["token_ms"]["split_side_stream_last_y"] = sum(to_y) / n
    out["token_ms"]["split_side_stream_total"] = sum(total) / n
    out["head_updates_per_token"] = units * layers
    assert A.stepq_device_error() == 0
    return out


def calib(name="pool", layers=None):
    """The calibration statistics of App. A.3 on the device: omega and ell over
    the calibration stream, then the candidate distortions of states sampled
    from the FP32 recurrence (twice for row units, with pivots held out)."""
    import time
    import torch
    dev = torch.device("cuda")
    wl = W.WORKLOADS[name]
    if layers is not None:
        wl = wl.replace(layers=layers)
    cfg = A.Config.from_workload(wl)
    wl1 = wl.replace(layers=1)
    A.calibrate(A.Config.from_workload(wl1), wl1, dev, seqs=2, steps=8, device_inputs=True)   # warm-up
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    st = A.calibrate(cfg, wl, dev, device_inputs=True)
    torch.cuda.synchronize()
    t = time.perf_counter() - t0
    assert A.stepq_device_error() == 0
    return {"metric": "calibration statistics on the device", "unit": "s", "value": t,
            "workload": f"{name}: {wl.layers} layers x {wl.hv} heads, {wl.calib_seqs} sequences x "
                        f"{wl.calib_steps} tokens, states sampled every {wl.calib_every} updates",
            "calibration_tokens": int(st.n_tokens), "sampled_states_per_layer": int(st.n_samples)}


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    sub = ap.add_subparsers(dest="what", required=True)
    r = sub.add_parser("rows")
    r.add_argument("--slots", type=int, default=1024)
    r.add_argument("--bits", type=int, default=6, choices=[4, 6])
    p = sub.add_parser("prefill")
    p.add_argument("--slots", type=int, default=128)
    p.add_argument("--tokens", type=int, default=512)
    p.add_argument("--workload", default="gqa", choices=["gqa", "channel", "pool"])
    cb = sub.add_parser("calib")
    cb.add_argument("--workload", default="pool", choices=["gqa", "channel", "pool", "drift"])
    sp = sub.add_parser("split")
    sp.add_argument("--slots", type=int, default=1024)
    sp.add_argument("--layers", type=int, default=16)
    args = ap.parse_args(argv)
    if args.what == "rows":
        res = rows(args.slots, args.bits)
    elif args.what == "split":
        res = split(args.slots, args.layers)
    elif args.what == "calib":
        res = calib(args.workload)
    else:
        res = prefill(args.slots, args.tokens, args.workload)
    print(json.dumps(res))


if __name__ == "__main__":
    main()
