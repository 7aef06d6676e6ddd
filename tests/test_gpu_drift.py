"""The drift workload (4 layers x 32 heads, per-key-channel gates, row units):
teacher-forced parity of every layer at 6 and 4 bits, and the free-running drift
measurement against the FP32-state recurrence on a short run."""
import math

import numpy as np
import pytest

import oracle as O
from paper_2609_38169_gb300 import api as A, drift, workloads as W

from gpu_helpers import Tally, compare_pools, compare_y, plans, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as T
    if not T.cuda.is_available():
        pytest.skip("no CUDA device")
    return T


@pytest.mark.parametrize("kw", [
    {},                                                   # @6, candidates {4,6,8}
    dict(nominal_bits=4, candidates=(2, 4, 6, 8)),        # @4
])
def test_drift_workload_all_layers(torch, kw):
    """App. C.3 steps 1-7 on every layer of the 4-layer channel-gate plan."""
    batch = 8
    wl = W.WORKLOADS["drift"].replace(batch=batch, **kw)
    cfg, plan, oplan, _ = plans(wl)
    mp = W.model_params(wl)
    slots = np.random.default_rng(3).permutation(wl.pool_slots)[:batch].astype(np.int32)
    (slots_d,) = to_dev(slots)
    pool_o = np.zeros(wl.pool_slots * oplan.slot_stride, np.uint8)
    for layer in range(wl.layers):
        O.pool_encode(oplan, pool_o, layer, slots, O.warmup_states(wl, layer, batch))
    pool_d = A.alloc_pool(plan, wl.pool_slots)
    t = Tally()
    for step in range(2):
        for layer in range(wl.layers):
            inp = W.step_inputs(wl, mp, W.STREAM_DECODE, step, layer, batch=batch)
            pool_d.copy_(torch.from_numpy(pool_o))
            q, k, v, beta, gate = to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate)
            y_d = torch.empty((batch, wl.hv, 128), dtype=torch.float32, device="cuda")
            A.stepq_decode_step(plan, layer, pool_d, slots_d, q, k, v, beta, gate, y_d)
            y_o = O.pool_step(oplan, pool_o, layer, slots, inp)
            compare_y(t, y_d.cpu().numpy(), y_o)
            compare_pools(t, pool_d.cpu().numpy(), pool_o, oplan, layer, slots)
    print(kw, t.summary())
    t.check()
    assert A.stepq_device_error() == 0


def test_drift_run_short(torch):
    """Free-running drift over 96 steps: finite, below the signal, and ordered by
    storage width (6-bit STEPQuant below 4-bit; INT8 below INT4)."""
    res = drift.run(steps=96, every=32, batch=8, warmup=8, calib=dict(seqs=2, steps=32))
    assert [r["step"] for r in res["records"]] == [32, 64, 96]
    last = res["records"][-1]
    for name in drift.VARIANTS:
        for key in ("at_step", "window_rms"):
            e = last[name][key]
            assert math.isfinite(e) and 0.0 < e < 1.0, (name, key, e)
    for r in res["records"]:
        assert r["stepq6"]["window_rms"] < r["stepq4"]["window_rms"]
        assert r["int8"]["window_rms"] < r["int4"]["window_rms"]
        assert r["stepq6"]["window_rms"] < r["int4"]["window_rms"]
    bpv = {n: v["bits_per_value"] for n, v in res["variants"].items()}
    assert 6.0 < bpv["stepq6"] < 6.6 and 4.0 < bpv["stepq4"] < 4.6
    assert 8.0 < bpv["int8"] < 8.2 and 4.0 < bpv["int4"] < 4.2


def test_drift_ablations_short(torch):
    """The component ablations of Sec. 5.4 run free for 32 steps: finite errors,
    6-bit below 4-bit for each ablation, and storage near the nominal width."""
    res = drift.run(steps=32, every=32, batch=4, warmup=8, variants=tuple(drift.ABLATIONS),
                    calib=dict(seqs=2, steps=32))
    last = res["records"][-1]
    for name in drift.ABLATIONS:
        e = last[name]["window_rms"]
        assert math.isfinite(e) and 0.0 < e < 1.0, (name, e)
    for a in ("spatial", "temporal", "temporal{}_nopiv", "stepq{}_nopiv"):
        n6, n4 = (a.format(6), a.format(4)) if "{}" in a else (a + "6", a + "4")
        assert last[n6]["window_rms"] < last[n4]["window_rms"]
    bpv = {n: v["bits_per_value"] for n, v in res["variants"].items()}
    for n, b in bpv.items():
        nominal = 6 if "6" in n else 4
        assert nominal < b < nominal + 0.6, (n, b)
