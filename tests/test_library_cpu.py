"""CPU-side checks of the C-ABI library (no GPU needed): it loads, exports every
symbol include/stepq.h declares, builds plans whose maps match the oracle's bit
for bit, and rejects bad arguments before launching anything."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2609_38169_gb300 import _lib, api as A, workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_symbols():
    src = open(os.path.join(ROOT, "include", "stepq.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return set(re.findall(r"\b(stepq_\w+)\s*\(", src))


def test_library_exports_every_declared_symbol():
    L = _lib.lib()
    declared = _declared_symbols()
    assert len(declared) >= 20
    for name in declared:
        assert hasattr(L, name), name
    assert declared == set(_lib.SIGNATURES), declared ^ set(_lib.SIGNATURES)
    assert A.version().startswith("stepq")


def _stats(oracle, wl, seqs=2, steps=24):
    return oracle.calibrate(wl, seqs=seqs, steps=steps)


@pytest.mark.parametrize("name,kw", [
    ("tiny", {}),
    ("gqa", {}),
    ("channel", {}),
    ("pool", dict(layers=2)),
    ("gqa", dict(n_pivots=3)),
    ("channel", dict(nominal_bits=6, candidates=(4, 6, 8), n_pivots=10)),
])
def test_plan_matches_oracle_bit_exact(oracle, name, kw):
    """Bit-allocation maps, pivots, layout offsets and slot stride are identical;
    w identical (both evaluate the footnote of Sec. 4.3 in fp64 and round once)."""
    wl = W.WORKLOADS[name].replace(**kw)
    st = _stats(oracle, wl, seqs=2, steps=16)
    ora = oracle.plan_from_stats(wl, st)
    cfg = A.Config.from_workload(wl)
    lib_piv = A.stepq_select_pivots(cfg, st.mean_log_ret, st.dist_stage1)
    assert np.array_equal(lib_piv, st.pivot)
    plan = A.stepq_fit_scales(cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
    assert np.array_equal(plan.unit_bits, ora.unit_bits)
    assert np.array_equal(plan.pivot_mask, ora.pivot)
    assert np.array_equal(plan.head_offset, ora.head_off)
    assert np.array_equal(plan.head_bytes, ora.head_bytes)
    assert plan.slot_stride == ora.slot_stride
    assert np.array_equal(plan.w, ora.w)
    assert np.allclose(plan.lifetime, ora.L, rtol=1e-15)
    # budget: pivots count as 8-bit replacements (App. D)
    n = plan.n_units
    assert np.sum(plan.unit_bits[plan.pivot_mask == 0]) + 8 * plan.pivot_mask.sum() <= wl.nominal_bits * n


def test_plan_without_given_pivots_selects_them(oracle):
    wl = W.WORKLOADS["gqa"].replace(n_pivots=4)
    st = _stats(oracle, wl, seqs=2, steps=16)
    cfg = A.Config.from_workload(wl)
    plan = A.stepq_fit_scales(cfg, st.omega, st.mean_log_ret, st.dist)
    assert np.array_equal(plan.pivot_mask, st.pivot)


def test_paper_shape_plan_bytes():
    """App. F.1: 29,999,104 B per request for 48 x 48 head units @6 with 32 pivots."""
    cfg = A.Config(n_layers=48, n_key_heads=16, n_value_heads=48, nominal_bits=6, n_pivots=32)
    n = A.stepq_num_units(cfg)
    rng = np.random.default_rng(3)
    d = np.sort(np.exp(rng.normal(0, 2, (n, 3))), axis=1)[:, ::-1]
    d = np.concatenate([d, 1e-9 * np.ones((n, 1))], axis=1)
    omega = np.exp(rng.normal(0, 1, (48, 48, 128))).astype(np.float32)
    plan = A.stepq_fit_scales(cfg, omega, rng.normal(-0.01, 0.003, n), d)
    assert plan.slot_stride == 29_999_104


@pytest.mark.parametrize("name,kw", [("gqa", dict(n_pivots=3)), ("channel", {}), ("pool", dict(layers=2))])
def test_temporal_slot_bytes(oracle, name, kw):
    """"Temporal only" layout (Sec. 5.4): per head s[128] fp16 plus 16 b_i bytes per
    row at the plan's widths (pivots 256 B), heads in (layer, head) order."""
    wl = W.WORKLOADS[name].replace(**kw)
    st = _stats(oracle, wl, seqs=1, steps=16)
    oplan = oracle.plan_from_stats(wl, st)
    cfg = A.Config.from_workload(wl)
    plan = A.stepq_fit_scales(cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
    total = sum(oracle.temporal_head_bytes(rb) for l in range(wl.layers)
                for rb in oplan.layer_row_bits(l))
    assert A.stepq_temporal_slot_bytes(plan) == (total + 255) // 256 * 256


def test_argument_errors_before_launch():
    L = _lib.lib()
    cfg = A.Config(n_layers=1, n_key_heads=4, n_value_heads=4).c()
    bad = A.Config(n_layers=1, n_key_heads=3, n_value_heads=4).c()
    assert L.stepq_num_units(C.byref(bad)) == 0
    h = C.c_void_p()
    assert L.stepq_fit_scales(C.byref(cfg), None, C.byref(h)) == 1          # STEPQ_ERR_ARG
    dk = A.Config(n_layers=1, n_key_heads=4, n_value_heads=4, dk=64).c()
    assert L.stepq_num_units(C.byref(dk)) == 0
    # null pool / plan
    assert L.stepq_decode_step(None, 0, None, 1, None, 1, None, None, None, None, None, None, None) == 1
    assert L.stepq_fp32_decode_step(C.byref(cfg), 5, C.c_void_p(256), 1, C.c_void_p(256), 1,
                                    None, None, None, None, None, None, None) == 1
    assert L.stepq_fp32_exact_read_step(C.byref(cfg), 0, C.c_void_p(256), None, 1, C.c_void_p(256), 1,
                                        None, None, C.c_void_p(256), None, None, C.c_void_p(256),
                                        None) == 1
    assert L.stepq_decode_readout(None, 0, None, 1, None, 1, None, None, None, None, None, None,
                                  None, None) == 1
    assert L.stepq_decode_writeback(None, 0, None, 1, None, 1, None, None, None, None, None) == 1
    assert L.stepq_intb_slot_bytes(C.byref(cfg), 3) == 0
    assert L.stepq_intb_slot_bytes(C.byref(cfg), 8) == (256 + 128 * 128) * 4
    assert L.stepq_intb_slot_bytes(C.byref(cfg), 6) == (256 + 128 * 96) * 4
    assert L.stepq_status_str(2) == b"slot id out of range"


def test_host_only_plan_refuses_device_calls(oracle):
    import torch
    if torch.cuda.is_available():
        pytest.skip("host-only plans exist only without a CUDA device")
    wl = W.WORKLOADS["tiny"]
    st = _stats(oracle, wl, seqs=1, steps=8)
    cfg = A.Config.from_workload(wl)
    plan = A.stepq_fit_scales(cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
    L = _lib.lib()
    fake = C.c_void_p(1 << 20)   # aligned, never dereferenced: the call must refuse first
    r = L.stepq_decode_step(plan.handle, 0, fake, 1, fake, 1, fake, fake, fake, fake, fake, fake, None)
    assert r == 5                                                             # STEPQ_ERR_CUDA


def test_drift_variants_and_cli():
    """The drift module's variant table and command line (no device work)."""
    from paper_2609_38169_gb300 import drift
    assert set(drift.VARIANTS) == {"stepq6", "stepq4", "int8", "int6", "int4"}
    assert drift.VARIANTS["stepq4"]["candidates"] == (2, 4, 6, 8)
    with pytest.raises(SystemExit) as e:
        drift.main(["--help"])
    assert e.value.code == 0


def test_feedback_cli():
    """The feedback-experiment module's command line (no device work)."""
    from paper_2609_38169_gb300 import feedback
    with pytest.raises(SystemExit) as e:
        feedback.main(["--help"])
    assert e.value.code == 0
    with pytest.raises(SystemExit) as e:
        feedback.main(["--codecs", "int5"])
    assert e.value.code == 2


def test_measure_cli():
    """The secondary-measurement module parses its subcommands (no device work)."""
    from paper_2609_38169_gb300 import measure
    for argv in (["--help"], ["rows", "--help"], ["prefill", "--help"], ["split", "--help"], ["calib", "--help"]):
        with pytest.raises(SystemExit) as e:
            measure.main(argv)
        assert e.value.code == 0
