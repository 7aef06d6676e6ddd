"""Long-generation drift of the compressed recurrent state against the FP32-state
recurrence (the drift workload: 4 layers x 32 heads with per-key-channel gates,
128 slots, 8192 decode steps).

Every variant starts from the same FP32 state (warm-up steps from zero on the
warm-up stream), is quantized once, and then runs free: each step reads its own
compressed state, updates it and writes it back (STEPQuant: App. C.3 steps 1-7;
uniform INT-b: the rowwise absmax codec of App. B.5; the component ablations of
Sec. 5.4, listed in ABLATIONS). The FP32-state kernel runs
beside them on identical inputs. Every `every` steps the relative readout error
||y - y_fp32|| / ||y_fp32|| over all layers, slots and heads is recorded, for
that step and as the RMS over the window since the previous record (the
paper's error-accumulation view, Prop. 1: a state error is carried forward by
the gates and corrected by the Delta rule's own retrieval).

Everything runs in the library's kernels; PyTorch only holds the buffers.
"""
from __future__ import annotations

import argparse
import json
import math
import sys
import time

from . import api as A, workloads as W

D = 128

# name -> how the variant stores the state
VARIANTS = {
    "stepq6": dict(kind="stepq", nominal_bits=6, candidates=(4, 6, 8)),
    "stepq4": dict(kind="stepq", nominal_bits=4, candidates=(2, 4, 6, 8)),
    "int8": dict(kind="intb", bits=8),
    "int6": dict(kind="intb", bits=6),
    "int4": dict(kind="intb", bits=4),
}
# Component ablations of Sec. 5.4: "Spatial only" is the dual-axis codec at one
# uniform width without pivots; "Temporal only" is the calibrated allocation
# with its FP16 pivots under the rowwise absmax quantizer of App. B.5, and
# "Temporal w/o pivots" the same without pivots. STEPQuant without its pivots
# is added beside them.
ABLATIONS = {
    "spatial6": dict(kind="stepq", nominal_bits=6, candidates=(6,), n_pivots=0),
    "spatial4": dict(kind="stepq", nominal_bits=4, candidates=(4,), n_pivots=0),
    "temporal6": dict(kind="temporal", nominal_bits=6, candidates=(4, 6, 8)),
    "temporal4": dict(kind="temporal", nominal_bits=4, candidates=(2, 4, 6, 8)),
    "temporal6_nopiv": dict(kind="temporal", nominal_bits=6, candidates=(4, 6, 8), n_pivots=0),
    "temporal4_nopiv": dict(kind="temporal", nominal_bits=4, candidates=(2, 4, 6, 8), n_pivots=0),
    "stepq6_nopiv": dict(kind="stepq", nominal_bits=6, candidates=(4, 6, 8), n_pivots=0),
    "stepq4_nopiv": dict(kind="stepq", nominal_bits=4, candidates=(2, 4, 6, 8), n_pivots=0),
}
ALL = {**VARIANTS, **ABLATIONS}


class _Variant:
    def __init__(self, name, spec, wl, slots, ref, device, calib):
        import torch
        self.name = name
        self.kind = spec["kind"]
        L = wl.layers
        if self.kind in ("stepq", "temporal"):
            wlv = wl.replace(nominal_bits=spec["nominal_bits"], candidates=spec["candidates"],
                             n_pivots=spec.get("n_pivots", wl.n_pivots))
            self.cfg = A.Config.from_workload(wlv)
            st = A.calibrate(self.cfg, wlv, device, device_inputs=True, **calib)
            self.plan = A.stepq_fit_scales(self.cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
        if self.kind == "stepq":
            self.pool = A.alloc_pool(self.plan, slots.numel(), device)
            A.stepq_quantize_pool(self.plan, -1, ref, slots, self.pool)
            self.slot_bytes = self.plan.slot_stride
        elif self.kind == "temporal":
            # dequantize, FP32 step, quantize, through a one-layer dense scratch
            self.slot_bytes = A.stepq_temporal_slot_bytes(self.plan)
            self.pool = torch.zeros(slots.numel() * self.slot_bytes, dtype=torch.uint8, device=device)
            A.stepq_temporal_quantize_pool(self.plan, -1, ref, slots, self.pool)
            self.cfg1 = A.Config.from_workload(wl.replace(layers=1))
            self.dense = torch.empty((slots.numel(), 1, wl.hv, D, D), dtype=torch.float32, device=device)
            self.dense_slots = torch.arange(slots.numel(), dtype=torch.int32, device=device)
        else:
            self.bits = spec["bits"]
            self.cfg = A.Config.from_workload(wl)
            self.slot_bytes = A.stepq_intb_slot_bytes(self.cfg, self.bits)
            self.pool = torch.zeros(slots.numel() * self.slot_bytes, dtype=torch.uint8, device=device)
            A.stepq_intb_quantize_pool(self.cfg, self.bits, -1, ref, slots, self.pool)
        self.bits_per_value = 8.0 * self.slot_bytes / (L * wl.hv * D * D)

    def step(self, layer, slots, q, k, v, beta, gate, y):
        if self.kind == "stepq":
            A.stepq_decode_step(self.plan, layer, self.pool, slots, q, k, v, beta, gate, y)
        elif self.kind == "temporal":
            A.stepq_temporal_dequantize_pool(self.plan, layer, self.pool, slots, self.dense)
            A.stepq_fp32_decode_step(self.cfg1, 0, self.dense, self.dense_slots, q, k, v, beta, gate, y)
            A.stepq_temporal_quantize_pool(self.plan, layer, self.dense, slots, self.pool)
        else:
            A.stepq_intb_decode_step(self.cfg, self.bits, layer, self.pool, slots, q, k, v, beta,
                                     gate, y)


def run(wl=None, steps=None, every=512, batch=None, variants=tuple(VARIANTS), warmup=None,
        calib=None, device="cuda", log=None) -> dict:
    """Free-running drift of each variant against the FP32-state kernel."""
    import torch
    wl = W.WORKLOADS["drift"] if wl is None else wl
    B = wl.batch if batch is None else batch
    wl = wl.replace(batch=B, pool_slots=B)
    steps = wl.steps if steps is None else steps
    warmup = wl.warmup_steps if warmup is None else warmup
    calib = {} if calib is None else calib
    dev = torch.device(device)
    L, Hv = wl.layers, wl.hv
    mp_dev = W.model_params_torch(W.model_params(wl), dev)
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    cfg = A.Config.from_workload(wl)

    ref = torch.zeros((B, L, Hv, D, D), dtype=torch.float32, device=dev)
    y_ref = torch.empty((L, B, Hv, D), dtype=torch.float32, device=dev)
    for t in range(warmup):
        for layer in range(L):
            inp = W.torch_step_inputs(wl, mp_dev, t, layer, dev, W.STREAM_WARMUP)
            A.stepq_fp32_decode_step(cfg, layer, ref, slots, *inp, y_ref[layer])
    vs = [_Variant(n, ALL[n], wl, slots, ref, dev, calib) for n in variants]
    ys = torch.empty((len(vs), L, B, Hv, D), dtype=torch.float32, device=dev)
    err_win = torch.zeros(len(vs), dtype=torch.float64, device=dev)
    ref_win = torch.zeros((), dtype=torch.float64, device=dev)
    records = []
    t0 = time.time()
    for t in range(steps):
        for layer in range(L):
            inp = W.torch_step_inputs(wl, mp_dev, t, layer, dev, W.STREAM_DECODE)
            A.stepq_fp32_decode_step(cfg, layer, ref, slots, *inp, y_ref[layer])
            for i, v in enumerate(vs):
                v.step(layer, slots, *inp, ys[i, layer])
        diff2 = (ys - y_ref[None]).double().square().sum(dim=(1, 2, 3, 4))
        ref2 = y_ref.double().square().sum()
        err_win += diff2
        ref_win += ref2
        if (t + 1) % every == 0 or t + 1 == steps:
            at = torch.sqrt(diff2 / ref2).cpu().tolist()
            win = torch.sqrt(err_win / ref_win).cpu().tolist()
            rec = {"step": t + 1}
            for i, v in enumerate(vs):
                rec[v.name] = {"at_step": at[i], "window_rms": win[i]}
            records.append(rec)
            err_win.zero_()
            ref_win.zero_()
            if log:
                log(f"step {t + 1:6d}  " + "  ".join(
                    f"{v.name} {at[i]:.3e}/{win[i]:.3e}" for i, v in enumerate(vs)) +
                    f"  ({time.time() - t0:.0f} s)")
    assert A.stepq_device_error() == 0
    return {
        "workload": f"{wl.name}: {L} layers x {Hv} heads, d_k=d_v=128, {B} slots, per-key-channel "
                    f"gates, {warmup} FP32 warm-up steps, {steps} decode steps, channel spreads "
                    f"k {wl.k_sigma} / v {wl.v_sigma}",
        "every": every,
        "variants": {v.name: {"bits_per_value": v.bits_per_value, "slot_bytes": v.slot_bytes}
                     for v in vs},
        "fp32_slot_bytes": L * Hv * D * D * 4,
        "records": records,
    }


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--every", type=int, default=512)
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--variants", default=",".join(VARIANTS),
                    help="comma list from " + ", ".join(ALL))
    ap.add_argument("--geometry", action="store_true",
                    help="key- and value-channel spreads sized to the paper's state geometry (App. B.6)")
    ap.add_argument("--out", default=None, help="write the JSON result here")
    args = ap.parse_args(argv)
    wl = W.WORKLOADS["drift"]
    if args.geometry:
        wl = W.with_geometry(wl)
    res = run(wl, steps=args.steps, every=args.every, batch=args.batch,
              variants=tuple(args.variants.split(",")),
              log=lambda s: print(s, file=sys.stderr, flush=True))
    text = json.dumps(res, indent=1)
    if args.out:
        with open(args.out, "w") as f:
            f.write(text)
    print(text)


if __name__ == "__main__":
    main()
