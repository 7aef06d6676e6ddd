"""ctypes declarations of libstepq.so (include/stepq.h). Marshalling only."""
from __future__ import annotations

import ctypes as C
import os

from . import build_ext

P = C.c_void_p
I = C.c_int
SZ = C.c_size_t


class StepqConfig(C.Structure):
    _fields_ = [("dk", I), ("dv", I), ("n_layers", I), ("n_key_heads", I), ("n_value_heads", I),
                ("gate_kind", I), ("nominal_bits", I), ("n_candidates", I),
                ("candidates", I * 4), ("n_pivots", I), ("horizon", I), ("fit_iters", I)]


class StepqCalib(C.Structure):
    _fields_ = [("omega", P), ("mean_log_ret", P), ("distortion", P), ("pivot_mask", P)]


class StepqCalibResult(C.Structure):
    _fields_ = [("omega", P), ("mean_log_ret", P), ("distortion", P), ("distortion_stage1", P),
                ("pivot_mask", P), ("n_tokens", I), ("n_samples", I)]


class StepqPlanInfo(C.Structure):
    _fields_ = [("slot_stride", SZ), ("n_units", SZ), ("unit_bits", P), ("pivot_mask", P),
                ("w", P), ("lifetime", P), ("head_offset", P), ("head_bytes", P)]


CFG = C.POINTER(StepqConfig)

# name -> (restype, argtypes); the exported symbol set of include/stepq.h
SIGNATURES = {
    "stepq_num_units": (SZ, [CFG]),
    "stepq_row_weights": (I, [CFG, P, P]),
    "stepq_lifetime_weight": (C.c_double, [C.c_double, I]),
    "stepq_select_pivots": (I, [CFG, P, P, P]),
    "stepq_fit_scales": (I, [CFG, C.POINTER(StepqCalib), C.POINTER(P)]),
    "stepq_plan_query": (I, [P, C.POINTER(StepqPlanInfo)]),
    "stepq_plan_destroy": (None, [P]),
    "stepq_quantize_pool": (I, [P, I, P, P, I, P, I, P]),
    "stepq_dequantize_pool": (I, [P, I, P, I, P, I, P, P]),
    "stepq_decode_readout": (I, [P, I, P, I, P, I, P, P, P, P, P, P, P, P]),
    "stepq_decode_writeback": (I, [P, I, P, I, P, I, P, P, P, P, P]),
    "stepq_temporal_slot_bytes": (SZ, [P]),
    "stepq_temporal_quantize_pool": (I, [P, I, P, P, I, P, I, P]),
    "stepq_temporal_dequantize_pool": (I, [P, I, P, I, P, I, P, P]),
    "stepq_decode_step": (I, [P, I, P, I, P, I, P, P, P, P, P, P, P]),
    "stepq_fp32_decode_step": (I, [CFG, I, P, I, P, I, P, P, P, P, P, P, P]),
    "stepq_prefill_fp32": (I, [CFG, I, I, P, P, P, P, P, P, P, P]),
    "stepq_fp32_exact_read_step": (I, [CFG, I, P, P, I, P, I, P, P, P, P, P, P, P]),
    "stepq_intb_slot_bytes": (SZ, [CFG, I]),
    "stepq_intb_quantize_pool": (I, [CFG, I, I, P, P, I, P, I, P]),
    "stepq_intb_dequantize_pool": (I, [CFG, I, I, P, I, P, I, P, P]),
    "stepq_intb_decode_step": (I, [CFG, I, I, P, I, P, I, P, P, P, P, P, P, P]),
    "stepq_calib_observe": (I, [CFG, I, P, P, P, P, I, P, P, P]),
    "stepq_calib_distortion": (I, [CFG, I, P, P, P, I, P, P]),
    "stepq_calib_workspace_bytes": (SZ, [CFG, I]),
    "stepq_debug_stall": (I, [C.c_longlong, I]),
    "stepq_calibrate_from_trace": (I, [CFG, I, I, I, P, P, P, P, P, P, SZ, C.POINTER(StepqCalibResult), P]),
    "stepq_validate_slots": (I, [P, I, I, P, P, P]),
    "stepq_validate_slots_noalloc": (I, [P, I, I, P, P]),
    "stepq_device_error": (I, [P]),
    "stepq_stream_status": (I, [P]),
    "stepq_status_str": (C.c_char_p, [I]),
    "stepq_version": (C.c_char_p, []),
}

_lib = None


def lib(build: bool = True):
    """Load libstepq.so (building it first if asked). Raises if it cannot be loaded:
    there is no fallback path."""
    global _lib
    if _lib is None:
        path = build_ext.build() if build else build_ext.SO
        if not os.path.exists(path):
            raise RuntimeError(f"libstepq.so not built at {path}")
        L = C.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


class StepqError(RuntimeError):
    def __init__(self, status: int, what: str):
        msg = lib().stepq_status_str(status).decode()
        super().__init__(f"{what}: {msg} (status {status})")
        self.status = status


def check(status: int, what: str):
    if status != 0:
        raise StepqError(status, what)
