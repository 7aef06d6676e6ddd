"""Single-injection feedback experiment (App. B.1) on the GPU against the oracle.

The device driver (`feedback.run`) and a plain oracle restatement of the same
experiment take the same seeded inputs; their per-trajectory error sums for
the native and the exact-read path agree to rounding.
"""
import numpy as np
import pytest

from paper_2609_38169_gb300 import feedback, workloads as W
from gpu_helpers import to_dev

import oracle as O

pytestmark = pytest.mark.gpu
D = 128


@pytest.fixture(scope="module")
def torch():
    import torch as T
    if not T.cuda.is_available():
        pytest.skip("no CUDA device")
    return T


def _oracle_experiment(wl, B, steps, inject, bits):
    mp = W.model_params(wl)
    ref = np.zeros((B, wl.hv, D, D), np.float32)
    nat = er = None
    e_nat = np.zeros(B)
    e_er = np.zeros(B)
    for t in range(steps):
        inp = W.step_inputs(wl, mp, W.STREAM_DECODE, t, 0, batch=B)
        args = (inp.q, inp.k, inp.v, inp.beta, inp.gate)
        if t >= inject:
            y_nat = O.delta_batch(nat, *args)
            y_er = O.delta_batch_read(er, ref, *args)
        y_ref = O.delta_batch(ref, *args)
        if t + 1 == inject:
            nat = np.stack([np.stack([O.intb_decode_head(O.intb_encode_head(ref[b, h], bits), bits)
                                      for h in range(wl.hv)]) for b in range(B)]).astype(np.float32)
            er = nat.copy()
        elif t >= inject:
            e_nat += ((y_nat.astype(np.float64) - y_ref) ** 2).sum(axis=(1, 2))
            e_er += ((y_er.astype(np.float64) - y_ref) ** 2).sum(axis=(1, 2))
    return e_nat, e_er


@pytest.mark.parametrize("name", ["gqa", "channel"])
def test_feedback_matches_oracle(torch, name):
    B, steps, inject = 2, 40, 8
    wl = W.WORKLOADS[name].replace(layers=1, batch=B, pool_slots=B)
    mp = W.model_params(wl)

    def inputs(t):
        inp = W.step_inputs(wl, mp, W.STREAM_DECODE, t, 0, batch=B)
        return to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate)

    res = feedback.run(wl, trajectories=B, steps=steps, inject=inject, codecs=("int6", "int8"),
                       every=16, inputs=inputs)
    for bits in (6, 8):
        e_nat, e_er = _oracle_experiment(wl, B, steps, inject, bits)
        r = res["codecs"][f"int{bits}"]
        assert np.allclose(r["native_per_trajectory"], e_nat, rtol=1e-3)
        assert np.allclose(r["exact_read_per_trajectory"], e_er, rtol=1e-3)
        assert r["native_sq_err"] > 0 and r["exact_read_sq_err"] > 0
    # INT6 injects a larger error than INT8 on both paths
    assert res["codecs"]["int6"]["native_sq_err"] > res["codecs"]["int8"]["native_sq_err"]
    assert res["windows"][-1]["after_step"] == steps
