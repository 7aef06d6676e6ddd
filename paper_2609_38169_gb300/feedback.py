"""Single-injection feedback experiment (App. B.1).

The FP32-state recurrence runs from a zero state. After `inject` updates its
state is quantized once (uniform INT-b, App. B.5, or a STEPQuant plan) and
dequantized, and two paths continue from that identical perturbed state with
no further quantization, on the reference's own inputs:

  native      the plain Delta step: the retrieval reads the path's own state,
              so the step removes the k-direction of the carried error,
              E_t = (I - beta k k^T) D_t E_{t-1} (Eq. self_correction);
  exact-read  the retrieval reads the reference state, u = k^T D S_ref, which
              leaves E_t = D_t E_{t-1}: the error only decays with the gates.

Each path's readout error against the reference is summed (squared) over
heads, trajectories (slots) and every step after the injection; the reported
ratio is exact-read over native, overall and per trajectory.

Everything runs in the library's kernels; PyTorch only holds the buffers.
"""
from __future__ import annotations

import argparse
import json
import sys
import time

from . import api as A, workloads as W

D = 128
CODECS = ("int6", "int8", "int4", "stepq6", "stepq4")


class _Injector:
    """Quantize-then-dequantize of a [B, 1, Hv, D, D] state with one codec."""

    def __init__(self, name, wl, slots, device, calib):
        import torch
        self.name = name
        if name.startswith("int"):
            self.bits = int(name[3:])
            self.cfg = A.Config.from_workload(wl)
            sb = A.stepq_intb_slot_bytes(self.cfg, self.bits)
            self.pool = torch.zeros(slots.numel() * sb, dtype=torch.uint8, device=device)
            self.slot_bytes = sb
        else:
            nb = int(name[5:])
            wlv = wl.replace(nominal_bits=nb, candidates=(4, 6, 8) if nb == 6 else (2, 4, 6, 8))
            self.cfg = A.Config.from_workload(wlv)
            st = A.calibrate(self.cfg, wlv, device, device_inputs=True, **calib)
            self.plan = A.stepq_fit_scales(self.cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
            self.pool = A.alloc_pool(self.plan, slots.numel(), device)
            self.slot_bytes = self.plan.slot_stride
        self.slots = slots

    def __call__(self, states, out):
        if hasattr(self, "plan"):
            A.stepq_quantize_pool(self.plan, -1, states, self.slots, self.pool)
            A.stepq_dequantize_pool(self.plan, -1, self.pool, self.slots, out)
        else:
            A.stepq_intb_quantize_pool(self.cfg, self.bits, -1, states, self.slots, self.pool)
            A.stepq_intb_dequantize_pool(self.cfg, self.bits, -1, self.pool, self.slots, out)


def run(wl=None, trajectories=4, steps=8192, inject=256, codecs=("int6", "int8"), every=512,
        inputs=None, calib=None, device="cuda", log=None) -> dict:
    """The matched single-injection experiment on one layer of `wl`.

    inputs(t) -> (q, k, v, beta, gate) device tensors for update t (default: the
    workload's device generator on the decode stream). Returns the error sums,
    their ratios and windowed sums every `every` steps after the injection.
    """
    import torch
    wl = W.WORKLOADS["gqa"] if wl is None else wl
    B = trajectories
    wl = wl.replace(layers=1, batch=B, pool_slots=B)
    if not 1 <= inject < steps:
        raise ValueError("need 1 <= inject < steps")
    dev = torch.device(device)
    if inputs is None:
        mp_dev = W.model_params_torch(W.model_params(wl), dev)
        inputs = lambda t: W.torch_step_inputs(wl, mp_dev, t, 0, dev, W.STREAM_DECODE)  # noqa: E731
    cfg = A.Config.from_workload(wl)
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    Hv = wl.hv
    inj = [_Injector(c, wl, slots, dev, {} if calib is None else calib) for c in codecs]
    nc = len(inj)
    ref = torch.zeros((B, 1, Hv, D, D), dtype=torch.float32, device=dev)
    # paths[c][0] native, paths[c][1] exact-read
    paths = torch.empty((nc, 2, B, 1, Hv, D, D), dtype=torch.float32, device=dev)
    y_ref = torch.empty((B, Hv, D), dtype=torch.float32, device=dev)
    ys = torch.empty((nc, 2, B, Hv, D), dtype=torch.float32, device=dev)
    err = torch.zeros((nc, 2, B), dtype=torch.float64, device=dev)
    win = torch.zeros((nc, 2), dtype=torch.float64, device=dev)
    ref2 = torch.zeros((), dtype=torch.float64, device=dev)
    windows = []
    t0 = time.time()
    for t in range(steps):
        q, k, v, beta, gate = inputs(t)
        if t >= inject:
            for c in range(nc):
                A.stepq_fp32_decode_step(cfg, 0, paths[c, 0], slots, q, k, v, beta, gate, ys[c, 0])
                A.stepq_fp32_exact_read_step(cfg, 0, paths[c, 1], ref, slots, q, k, v, beta, gate,
                                             ys[c, 1])
        A.stepq_fp32_decode_step(cfg, 0, ref, slots, q, k, v, beta, gate, y_ref)
        if t + 1 == inject:
            for c in range(nc):
                inj[c](ref, paths[c, 0])
                paths[c, 1].copy_(paths[c, 0])
        elif t >= inject:
            d2 = (ys - y_ref[None, None]).double().square().sum(dim=(-1, -2))
            err += d2
            win += d2.sum(dim=-1)
            ref2 += y_ref.double().square().sum()
            n = t + 1 - inject
            if n % every == 0 or t + 1 == steps:
                w = win.cpu().tolist()
                windows.append({"after_step": t + 1,
                                **{inj[c].name: {"native": w[c][0], "exact_read": w[c][1]}
                                   for c in range(nc)}})
                win.zero_()
                if log:
                    log(f"step {t + 1:6d}  " + "  ".join(
                        f"{inj[c].name} {w[c][0]:.3e}/{w[c][1]:.3e}" for c in range(nc)) +
                        f"  ({time.time() - t0:.0f} s)")
    assert A.stepq_device_error() == 0
    e = err.cpu().numpy()
    out = {
        "workload": f"{wl.name}: {Hv} heads ({wl.gate} gates), {B} trajectories, {steps} updates, "
                    f"one injection after update {inject}, {steps - inject} readouts compared, "
                    f"channel spreads k {wl.k_sigma} / v {wl.v_sigma}",
        "reference_sq_sum": float(ref2.cpu()),
        "codecs": {},
        "windows": windows,
    }
    for c in range(nc):
        nat, er = e[c, 0], e[c, 1]
        out["codecs"][inj[c].name] = {
            "native_sq_err": float(nat.sum()), "exact_read_sq_err": float(er.sum()),
            "ratio": float(er.sum() / nat.sum()) if nat.sum() > 0 else None,
            "ratio_per_trajectory": [float(a / b) if b > 0 else None for a, b in zip(er, nat)],
            "native_per_trajectory": nat.tolist(), "exact_read_per_trajectory": er.tolist(),
            "slot_bytes": inj[c].slot_bytes,
        }
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--trajectories", type=int, default=4)
    ap.add_argument("--steps", type=int, default=8192)
    ap.add_argument("--inject", type=int, default=256)
    ap.add_argument("--every", type=int, default=512)
    ap.add_argument("--workload", default="gqa", choices=["gqa", "channel"])
    ap.add_argument("--codecs", default="int6,int8", help="comma list from " + ", ".join(CODECS))
    ap.add_argument("--geometry", action="store_true",
                    help="key- and value-channel spreads sized to the paper's state geometry (App. B.6)")
    ap.add_argument("--out", default=None, help="write the JSON result here")
    args = ap.parse_args(argv)
    codecs = tuple(args.codecs.split(","))
    for c in codecs:
        if c not in CODECS:
            ap.error(f"unknown codec {c}")
    wl = W.WORKLOADS[args.workload]
    if args.geometry:
        wl = W.with_geometry(wl)
    res = run(wl, args.trajectories, args.steps, args.inject, codecs,
              args.every, log=lambda s: print(s, file=sys.stderr, flush=True))
    text = json.dumps(res, indent=1)
    if args.out:
        with open(args.out, "w") as f:
            f.write(text)
    print(text)


if __name__ == "__main__":
    main()
