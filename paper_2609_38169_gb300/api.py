"""Python binding of libstepq.so with the C entry points' names.

Arguments are marshalled (torch CUDA tensors -> device pointers, numpy arrays ->
host pointers); every computation runs in the library. A missing or unloadable
library raises: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass, field

import numpy as np

from . import _lib
from ._lib import StepqCalib, StepqConfig, StepqPlanInfo, check

D = 128
GATE_SCALAR = 0
GATE_CHANNEL = 1
PIVOT_BITS = 16


@dataclass
class Config:
    n_layers: int
    n_key_heads: int
    n_value_heads: int
    gate_kind: int = GATE_SCALAR
    nominal_bits: int = 6
    candidates: tuple = (4, 6, 8)
    n_pivots: int = 0
    horizon: int = 2048
    fit_iters: int = 1
    dk: int = D
    dv: int = D

    def c(self) -> StepqConfig:
        cs = list(self.candidates) + [0] * (4 - len(self.candidates))
        return StepqConfig(self.dk, self.dv, self.n_layers, self.n_key_heads, self.n_value_heads,
                           self.gate_kind, self.nominal_bits, len(self.candidates),
                           (C.c_int * 4)(*cs), self.n_pivots, self.horizon, self.fit_iters)

    @classmethod
    def from_workload(cls, wl, **kw) -> "Config":
        base = dict(n_layers=wl.layers, n_key_heads=wl.hk, n_value_heads=wl.hv,
                    gate_kind=GATE_SCALAR if wl.gate == "scalar" else GATE_CHANNEL,
                    nominal_bits=wl.nominal_bits, candidates=tuple(wl.candidates),
                    n_pivots=wl.n_pivots, horizon=wl.horizon, fit_iters=wl.fit_iters)
        base.update(kw)
        return cls(**base)

    @property
    def unit_rows(self) -> bool:
        return self.gate_kind == GATE_CHANNEL


class _Ptr(C.c_void_p):
    """A pointer argument that keeps its numpy array alive until the call returns."""
    __slots__ = ("_keep",)


def _np_ptr(a: np.ndarray | None):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"]
    ptr = _Ptr(a.ctypes.data)
    ptr._keep = a
    return ptr


def _dev_ptr(t, dtype=None):
    """Device pointer of a contiguous CUDA tensor (None passes through)."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"expected {dtype}, got {t.dtype}")
    return t.data_ptr()


def _stream(stream):
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return C.c_void_p(s.cuda_stream)


def version() -> str:
    return _lib.lib().stepq_version().decode()


# ------------------------------------------------------------------ plan
def stepq_num_units(cfg: Config) -> int:
    c = cfg.c()
    return _lib.lib().stepq_num_units(C.byref(c))


def stepq_row_weights(cfg: Config, omega: np.ndarray) -> np.ndarray:
    om = np.ascontiguousarray(omega, np.float32)
    w = np.zeros_like(om)
    c = cfg.c()
    check(_lib.lib().stepq_row_weights(C.byref(c), _np_ptr(om), _np_ptr(w)), "stepq_row_weights")
    return w


def stepq_lifetime_weight(ell: float, horizon: int) -> float:
    return _lib.lib().stepq_lifetime_weight(float(ell), int(horizon))


def stepq_select_pivots(cfg: Config, mean_log_ret, distortion) -> np.ndarray:
    c = cfg.c()
    n = stepq_num_units(cfg)
    lr = np.ascontiguousarray(mean_log_ret, np.float64).reshape(n)
    d = np.ascontiguousarray(distortion, np.float64).reshape(n, len(cfg.candidates) + 1)
    out = np.zeros(n, np.uint8)
    check(_lib.lib().stepq_select_pivots(C.byref(c), _np_ptr(lr), _np_ptr(d), _np_ptr(out)),
          "stepq_select_pivots")
    return out


class Plan:
    """A frozen plan (owned by the library; destroyed with this object)."""

    def __init__(self, cfg: Config, handle: int):
        self.cfg = cfg
        self._h = C.c_void_p(handle)
        info = StepqPlanInfo()
        check(_lib.lib().stepq_plan_query(self._h, C.byref(info)), "stepq_plan_query")
        n, L, Hv = info.n_units, cfg.n_layers, cfg.n_value_heads

        def view(ptr, ctype, count, dtype):
            return np.ctypeslib.as_array(C.cast(ptr, C.POINTER(ctype)), shape=(count,)).astype(dtype)

        self.slot_stride = int(info.slot_stride)
        self.n_units = int(n)
        self.unit_bits = view(info.unit_bits, C.c_int8, n, np.int8)
        self.pivot_mask = view(info.pivot_mask, C.c_uint8, n, np.uint8)
        self.w = view(info.w, C.c_float, L * Hv * D, np.float32).reshape(L, Hv, D)
        self.lifetime = view(info.lifetime, C.c_double, n, np.float64)
        self.head_offset = view(info.head_offset, C.c_uint64, L * Hv, np.uint64)
        self.head_bytes = view(info.head_bytes, C.c_uint32, L * Hv, np.uint32)

    @property
    def handle(self):
        return self._h

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value:
            try:
                _lib.lib(build=False).stepq_plan_destroy(h)
            except Exception:
                pass
            self._h = C.c_void_p(0)

    def pool_bytes(self, pool_slots: int) -> int:
        return pool_slots * self.slot_stride


def stepq_fit_scales(cfg: Config, omega, mean_log_ret, distortion, pivot_mask=None) -> Plan:
    c = cfg.c()
    n = stepq_num_units(cfg)
    om = np.ascontiguousarray(omega, np.float32)
    lr = np.ascontiguousarray(mean_log_ret, np.float64).reshape(n)
    d = np.ascontiguousarray(distortion, np.float64).reshape(n, len(cfg.candidates) + 1)
    pm = None if pivot_mask is None else np.ascontiguousarray(pivot_mask, np.uint8).reshape(n)
    cal = StepqCalib(_np_ptr(om), _np_ptr(lr), _np_ptr(d), _np_ptr(pm))
    h = C.c_void_p()
    check(_lib.lib().stepq_fit_scales(C.byref(c), C.byref(cal), C.byref(h)), "stepq_fit_scales")
    return Plan(cfg, h.value)


# ------------------------------------------------------------------ device path
def _pool_slots(pool, stride, pool_slots):
    if pool_slots is not None:
        return int(pool_slots)
    return int(pool.numel() * pool.element_size() // stride)


def alloc_pool(plan: Plan, pool_slots: int, device="cuda"):
    import torch
    return torch.zeros(plan.pool_bytes(pool_slots), dtype=torch.uint8, device=device)


def stepq_quantize_pool(plan: Plan, layer: int, states, slots, pool, pool_slots=None, stream=None):
    import torch
    B = slots.numel()
    check(_lib.lib().stepq_quantize_pool(plan.handle, layer, _dev_ptr(states, torch.float32),
                                         _dev_ptr(slots, torch.int32), B, _dev_ptr(pool),
                                         _pool_slots(pool, plan.slot_stride, pool_slots),
                                         _stream(stream)), "stepq_quantize_pool")


def stepq_dequantize_pool(plan: Plan, layer: int, pool, slots, states_out, pool_slots=None,
                          stream=None):
    import torch
    B = slots.numel()
    check(_lib.lib().stepq_dequantize_pool(plan.handle, layer, _dev_ptr(pool),
                                           _pool_slots(pool, plan.slot_stride, pool_slots),
                                           _dev_ptr(slots, torch.int32), B,
                                           _dev_ptr(states_out, torch.float32), _stream(stream)),
          "stepq_dequantize_pool")


def stepq_temporal_slot_bytes(plan: Plan) -> int:
    return int(_lib.lib().stepq_temporal_slot_bytes(plan.handle))


def stepq_temporal_quantize_pool(plan: Plan, layer: int, states, slots, pool, pool_slots=None,
                                 stream=None):
    import torch
    stride = stepq_temporal_slot_bytes(plan)
    check(_lib.lib().stepq_temporal_quantize_pool(plan.handle, layer, _dev_ptr(states, torch.float32),
                                                  _dev_ptr(slots, torch.int32), slots.numel(),
                                                  _dev_ptr(pool), _pool_slots(pool, stride, pool_slots),
                                                  _stream(stream)), "stepq_temporal_quantize_pool")


def stepq_temporal_dequantize_pool(plan: Plan, layer: int, pool, slots, states_out, pool_slots=None,
                                   stream=None):
    import torch
    stride = stepq_temporal_slot_bytes(plan)
    check(_lib.lib().stepq_temporal_dequantize_pool(plan.handle, layer, _dev_ptr(pool),
                                                    _pool_slots(pool, stride, pool_slots),
                                                    _dev_ptr(slots, torch.int32), slots.numel(),
                                                    _dev_ptr(states_out, torch.float32),
                                                    _stream(stream)), "stepq_temporal_dequantize_pool")


def stepq_decode_step(plan: Plan, layer: int, pool, slots, q, k, v, beta, gate, y,
                      pool_slots=None, stream=None):
    import torch
    f = torch.float32
    B = slots.numel()
    check(_lib.lib().stepq_decode_step(plan.handle, layer, _dev_ptr(pool),
                                       _pool_slots(pool, plan.slot_stride, pool_slots),
                                       _dev_ptr(slots, torch.int32), B, _dev_ptr(q, f),
                                       _dev_ptr(k, f), _dev_ptr(v, f), _dev_ptr(beta, f),
                                       _dev_ptr(gate, f), _dev_ptr(y, f), _stream(stream)),
          "stepq_decode_step")


def stepq_decode_readout(plan: Plan, layer: int, pool, slots, q, k, v, beta, gate, y, delta,
                         pool_slots=None, stream=None):
    import torch
    f = torch.float32
    check(_lib.lib().stepq_decode_readout(plan.handle, layer, _dev_ptr(pool),
                                          _pool_slots(pool, plan.slot_stride, pool_slots),
                                          _dev_ptr(slots, torch.int32), slots.numel(),
                                          _dev_ptr(q, f), _dev_ptr(k, f), _dev_ptr(v, f),
                                          _dev_ptr(beta, f), _dev_ptr(gate, f), _dev_ptr(y, f),
                                          _dev_ptr(delta, f), _stream(stream)),
          "stepq_decode_readout")


def stepq_decode_writeback(plan: Plan, layer: int, pool, slots, k, beta, gate, delta,
                           pool_slots=None, stream=None):
    import torch
    f = torch.float32
    check(_lib.lib().stepq_decode_writeback(plan.handle, layer, _dev_ptr(pool),
                                            _pool_slots(pool, plan.slot_stride, pool_slots),
                                            _dev_ptr(slots, torch.int32), slots.numel(),
                                            _dev_ptr(k, f), _dev_ptr(beta, f), _dev_ptr(gate, f),
                                            _dev_ptr(delta, f), _stream(stream)),
          "stepq_decode_writeback")


def stepq_fp32_decode_step(cfg: Config, layer: int, pool, slots, q, k, v, beta, gate, y,
                           pool_slots=None, stream=None):
    import torch
    f = torch.float32
    c = cfg.c()
    ps = pool_slots if pool_slots is not None else pool.shape[0]
    check(_lib.lib().stepq_fp32_decode_step(C.byref(c), layer, _dev_ptr(pool, f), int(ps),
                                            _dev_ptr(slots, torch.int32), slots.numel(),
                                            _dev_ptr(q, f), _dev_ptr(k, f), _dev_ptr(v, f),
                                            _dev_ptr(beta, f), _dev_ptr(gate, f), _dev_ptr(y, f),
                                            _stream(stream)), "stepq_fp32_decode_step")


def stepq_fp32_exact_read_step(cfg: Config, layer: int, pool, read_pool, slots, q, k, v, beta, gate,
                               y, pool_slots=None, stream=None):
    import torch
    f = torch.float32
    c = cfg.c()
    ps = pool_slots if pool_slots is not None else pool.shape[0]
    check(_lib.lib().stepq_fp32_exact_read_step(C.byref(c), layer, _dev_ptr(pool, f),
                                                _dev_ptr(read_pool, f), int(ps),
                                                _dev_ptr(slots, torch.int32), slots.numel(),
                                                _dev_ptr(q, f), _dev_ptr(k, f), _dev_ptr(v, f),
                                                _dev_ptr(beta, f), _dev_ptr(gate, f), _dev_ptr(y, f),
                                                _stream(stream)), "stepq_fp32_exact_read_step")


def stepq_prefill_fp32(cfg: Config, states, q, k, v, beta, gate, y, stream=None):
    """Chunked prefill over T tokens on FP32 states [B][Hv][128][128] (in place);
    q, k [B][T][Hk][128], v [B][T][Hv][128], beta [B][T][Hv], gate [B][T][Hv]
    or [B][T][Hv][128], y [B][T][Hv][128] out."""
    import torch
    f = torch.float32
    c = cfg.c()
    B, T = int(q.shape[0]), int(q.shape[1])
    check(_lib.lib().stepq_prefill_fp32(C.byref(c), B, T, _dev_ptr(states, f), _dev_ptr(q, f),
                                        _dev_ptr(k, f), _dev_ptr(v, f), _dev_ptr(beta, f),
                                        _dev_ptr(gate, f), _dev_ptr(y, f), _stream(stream)),
          "stepq_prefill_fp32")


def stepq_intb_slot_bytes(cfg: Config, bits: int) -> int:
    c = cfg.c()
    return int(_lib.lib().stepq_intb_slot_bytes(C.byref(c), bits))


def stepq_intb_quantize_pool(cfg: Config, bits: int, layer: int, states, slots, pool,
                             pool_slots=None, stream=None):
    import torch
    c = cfg.c()
    ps = _pool_slots(pool, stepq_intb_slot_bytes(cfg, bits), pool_slots)
    check(_lib.lib().stepq_intb_quantize_pool(C.byref(c), bits, layer,
                                              _dev_ptr(states, torch.float32),
                                              _dev_ptr(slots, torch.int32), slots.numel(),
                                              _dev_ptr(pool), ps, _stream(stream)),
          "stepq_intb_quantize_pool")


def stepq_intb_dequantize_pool(cfg: Config, bits: int, layer: int, pool, slots, states_out,
                               pool_slots=None, stream=None):
    import torch
    c = cfg.c()
    ps = _pool_slots(pool, stepq_intb_slot_bytes(cfg, bits), pool_slots)
    check(_lib.lib().stepq_intb_dequantize_pool(C.byref(c), bits, layer, _dev_ptr(pool), ps,
                                                _dev_ptr(slots, torch.int32), slots.numel(),
                                                _dev_ptr(states_out, torch.float32),
                                                _stream(stream)), "stepq_intb_dequantize_pool")


def stepq_intb_decode_step(cfg: Config, bits: int, layer: int, pool, slots, q, k, v, beta, gate,
                           y, pool_slots=None, stream=None):
    import torch
    f = torch.float32
    c = cfg.c()
    ps = _pool_slots(pool, stepq_intb_slot_bytes(cfg, bits), pool_slots)
    check(_lib.lib().stepq_intb_decode_step(C.byref(c), bits, layer, _dev_ptr(pool), ps,
                                            _dev_ptr(slots, torch.int32), slots.numel(),
                                            _dev_ptr(q, f), _dev_ptr(k, f), _dev_ptr(v, f),
                                            _dev_ptr(beta, f), _dev_ptr(gate, f), _dev_ptr(y, f),
                                            _stream(stream)), "stepq_intb_decode_step")


def stepq_calib_observe(cfg: Config, layer: int, q, k, beta, gate, omega_sum, logret_sum,
                        stream=None):
    import torch
    f = torch.float32
    c = cfg.c()
    check(_lib.lib().stepq_calib_observe(C.byref(c), layer, _dev_ptr(q, f), _dev_ptr(k, f),
                                         _dev_ptr(beta, f), _dev_ptr(gate, f), q.shape[0],
                                         _dev_ptr(omega_sum, torch.float64),
                                         _dev_ptr(logret_sum, torch.float64), _stream(stream)),
          "stepq_calib_observe")


def stepq_calib_distortion(cfg: Config, layer: int, w, pivot_rows, states, acc, stream=None):
    import torch
    c = cfg.c()
    check(_lib.lib().stepq_calib_distortion(C.byref(c), layer, _dev_ptr(w, torch.float32),
                                            _dev_ptr(pivot_rows, torch.uint8),
                                            _dev_ptr(states, torch.float32), states.shape[0],
                                            _dev_ptr(acc, torch.float64), _stream(stream)),
          "stepq_calib_distortion")


def stepq_validate_slots(slots, pool_slots: int, scratch, status_out, stream=None):
    import torch
    check(_lib.lib().stepq_validate_slots(_dev_ptr(slots, torch.int32), slots.numel(),
                                          int(pool_slots), _dev_ptr(scratch, torch.int32),
                                          _dev_ptr(status_out, torch.int32), _stream(stream)),
          "stepq_validate_slots")


def stepq_validate_slots_noalloc(slots, pool_slots: int, status_out, stream=None):
    """stepq_validate_slots without a scratch argument: the library keeps the
    bitmap in a fixed device array (pool_slots <= 1,048,576) and allocates nothing."""
    import torch
    check(_lib.lib().stepq_validate_slots_noalloc(_dev_ptr(slots, torch.int32), slots.numel(),
                                                  int(pool_slots),
                                                  _dev_ptr(status_out, torch.int32),
                                                  _stream(stream)),
          "stepq_validate_slots_noalloc")


def stepq_debug_stall(wait_cycles: int = 2_000_000_000, withhold_item: int = -1):
    """Test support: the wait bound of the pipelined decode kernels and an item
    whose copies never start (stepq_debug_stall; -1 = none). Defaults restore
    normal operation."""
    check(_lib.lib().stepq_debug_stall(int(wait_cycles), int(withhold_item)), "stepq_debug_stall")


def stepq_device_error(stream=None) -> int:
    return int(_lib.lib().stepq_device_error(_stream(stream)))


def stepq_stream_status(stream=None) -> int:
    return int(_lib.lib().stepq_stream_status(_stream(stream)))


# ------------------------------------------------------------------ calibration driver
@dataclass
class CalibStats:
    omega: np.ndarray
    mean_log_ret: np.ndarray
    dist_stage1: np.ndarray
    dist: np.ndarray
    pivot: np.ndarray
    n_tokens: int = 0
    n_samples: int = 0
    extra: dict = field(default_factory=dict)


def stepq_calibrate_from_trace(cfg: Config, q, k, v, beta, gate, every: int, stream=None) -> CalibStats:
    """The calibration protocol of App. A.3 on a device trace (q, k [L][T][n][Hk][128],
    v [L][T][n][Hv][128], beta [L][T][n][Hv], gate [L][T][n][Hv] or [L][T][n][Hv][128]),
    all in the library (stepq_calibrate_from_trace); the workspace comes from torch."""
    import torch
    f = torch.float32
    L, T, n = q.shape[0], q.shape[1], q.shape[2]
    c = cfg.c()
    lib = _lib.lib()
    nbytes = lib.stepq_calib_workspace_bytes(C.byref(c), n)
    if nbytes == 0:
        raise ValueError("invalid configuration or sequence count")
    ws = torch.empty(nbytes + 256, dtype=torch.uint8, device=q.device)
    base = (ws.data_ptr() + 255) // 256 * 256
    U = stepq_num_units(cfg)
    K1 = len(cfg.candidates) + 1
    omega = np.zeros((cfg.n_layers, cfg.n_value_heads, D), np.float32)
    ell = np.zeros(U, np.float64)
    dist = np.zeros((U, K1), np.float64)
    dist1 = np.zeros((U, K1), np.float64)
    pivot = np.zeros(U, np.uint8)
    res = _lib.StepqCalibResult(omega.ctypes.data, ell.ctypes.data, dist.ctypes.data, dist1.ctypes.data,
                                pivot.ctypes.data, 0, 0)
    check(lib.stepq_calibrate_from_trace(C.byref(c), n, T, int(every), _dev_ptr(q, f), _dev_ptr(k, f),
                                         _dev_ptr(v, f), _dev_ptr(beta, f), _dev_ptr(gate, f),
                                         C.c_void_p(base), nbytes, C.byref(res), _stream(stream)),
          "stepq_calibrate_from_trace")
    return CalibStats(omega, ell, dist1, dist, pivot, res.n_tokens, res.n_samples)


def calibrate(cfg: Config, wl, device="cuda", seqs=None, steps=None, every=None,
              device_inputs: bool = False) -> CalibStats:
    """Calibration statistics for `cfg` on the workload's calibration stream
    (App. A.3): the trace of `steps` tokens for `seqs` sequences per layer is
    drawn (on the GPU with `device_inputs`, else with the numpy generator the
    oracle shares) and handed to stepq_calibrate_from_trace, which does every
    step of the protocol."""
    import torch
    from . import workloads as W
    seqs = wl.calib_seqs if seqs is None else seqs
    steps = wl.calib_steps if steps is None else steps
    every = wl.calib_every if every is None else every
    mp = W.model_params(wl)
    dev = torch.device(device)
    mp_dev = W.model_params_torch(mp, dev) if device_inputs else None

    def inputs(t, layer):
        if device_inputs:
            return list(W.torch_step_inputs(wl, mp_dev, t, layer, dev, W.STREAM_CALIB, batch=seqs))
        inp = W.step_inputs(wl, mp, W.STREAM_CALIB, t, layer, batch=seqs)
        return [torch.from_numpy(a).to(dev) for a in (inp.q, inp.k, inp.v, inp.beta, inp.gate)]

    trace = None
    for layer in range(cfg.n_layers):
        for t in range(steps):
            xs = inputs(t, layer)
            if trace is None:
                trace = [torch.empty((cfg.n_layers, steps) + tuple(x.shape), dtype=torch.float32, device=dev)
                         for x in xs]
            for dst, x in zip(trace, xs):
                dst[layer, t].copy_(x)
    return stepq_calibrate_from_trace(cfg, *trace, every=every)
