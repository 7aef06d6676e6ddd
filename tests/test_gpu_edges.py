"""Edge cases of the decode path against the oracle (App. C.3 steps 1-7):
degenerate states and the largest head count a launch accepts.

States: an all-zero state (every scale at its FP16 floor, codes 0), states
scaled by 1e9 (the clip-free column start exceeds the FP16 range, so the
codes take the clamped path), states scaled by 1e-12 (row factors at the
FP16 floor) and a state of tiny values with a few large outliers. Each runs
two teacher-forced decode steps under the parity rules of gpu_helpers, with
one addition for FP16 pivot values: the tile is fp32 (the oracle rounds an
fp64 result once), so a pivot value that is the small difference of large
terms (the retrieval's sum, the update's two parts) may differ by the fp32
rounding of those terms, 2^-21 of their magnitude, even when that exceeds one
FP16 ulp of the result.
"""
import numpy as np
import pytest

import oracle as O
from paper_2609_38169_gb300 import api as A, workloads as W

from gpu_helpers import Tally, compare_pools, compare_y, plans, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as T
    if not T.cuda.is_available():
        pytest.skip("no CUDA device")
    return T


def _degenerate_states(wl, B=4):
    base = W.random_states(wl, B * wl.hv, seed=21).reshape(B, wl.hv, 128, 128).astype(np.float64)
    S = np.zeros_like(base)                                   # slot 0: zero state
    S[1] = base[1] * 1e9                                      # slot 1: huge
    S[2] = base[2] * 1e-12                                    # slot 2: tiny
    S[3] = base[3] * 1e-6                                     # slot 3: tiny with outliers
    rng = np.random.default_rng(5)
    for h in range(wl.hv):
        idx = rng.integers(0, 128, size=(3, 2))
        S[3, h, idx[:, 0], idx[:, 1]] = rng.choice([-1.0, 1.0], 3) * 1e3
    return S.astype(np.float32)


def _update_term_bound(wl, S_hat, inp):
    """Absolute fp32 rounding allowance of the updated state X = D S + beta k
    (v - k^T D S)^T: 2^-21 of the magnitudes that enter it, |D S_ij| +
    |beta k_i| (|v_j| + sum_i' |k_i' (D S)_i'j|); the retrieval's fp32 sum
    carries the rounding of its largest terms into delta_j, and the update's
    terms may nearly cancel. S_hat: [B][Hv][128][128] decoded state."""
    grp = wl.hv // wl.hk
    k = np.repeat(inp.k.astype(np.float64), grp, axis=1)
    g = inp.gate.astype(np.float64)
    g = g if g.ndim == 3 else np.broadcast_to(g[..., None], k.shape)
    DS = g[..., None] * S_hat
    dmag = np.abs(inp.v.astype(np.float64)) + np.einsum("bhi,bhij->bhj", np.abs(k), np.abs(DS))
    T = np.abs(DS) + np.abs(inp.beta.astype(np.float64)[..., None, None] * k[..., None]) * dmag[:, :, None, :]
    return 2.0 ** -21 * T


def _teacher_forced(torch, wl, S, steps=2):
    cfg, plan, oplan, _ = plans(wl)
    mp = W.model_params(wl)
    B = S.shape[0]
    slots = np.arange(B, dtype=np.int32)[::-1].copy()
    pool_o = np.zeros(wl.pool_slots * oplan.slot_stride, np.uint8)
    O.pool_encode(oplan, pool_o, 0, slots, S)
    pool_d = A.alloc_pool(plan, wl.pool_slots)
    (slots_d, S_d) = to_dev(slots, S)
    A.stepq_quantize_pool(plan, 0, S_d, slots_d, pool_d)
    t = Tally()
    compare_pools(t, pool_d.cpu().numpy(), pool_o, oplan, 0, slots)
    for step in range(steps):
        inp = W.step_inputs(wl, mp, W.STREAM_DECODE, step, 0, batch=B)
        pool_d.copy_(torch.from_numpy(pool_o))
        tol = _update_term_bound(wl, O.pool_decode(oplan, pool_o, 0, slots).astype(np.float64), inp)
        q, k, v, beta, gate = to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate)
        y_d = torch.empty((B, wl.hv, 128), dtype=torch.float32, device="cuda")
        A.stepq_decode_step(plan, 0, pool_d, slots_d, q, k, v, beta, gate, y_d)
        y_o = O.pool_step(oplan, pool_o, 0, slots, inp)
        assert np.isfinite(y_d.cpu().numpy()).all()
        compare_y(t, y_d.cpu().numpy(), y_o)
        compare_pools(t, pool_d.cpu().numpy(), pool_o, oplan, 0, slots, piv_tol=tol)
    return t


@pytest.mark.parametrize("name,kw", [("gqa", dict(n_pivots=3, pool_slots=4)),
                                     ("channel", dict(pool_slots=4))])
def test_degenerate_states(torch, name, kw):
    wl = W.WORKLOADS[name].replace(**kw)
    t = _teacher_forced(torch, wl, _degenerate_states(wl))
    print(name, t.summary())
    t.check()
    assert A.stepq_device_error() == 0


@pytest.mark.parametrize("bits,name", [(8, "gqa"), (4, "channel")])
def test_intb_degenerate_states(torch, bits, name):
    """The INT-b comparison kernel on the same edge-case states: a zero state,
    a huge one whose row scales are capped at 65504 (so the codes are clamped
    to +-q_b, App. B.5), tiny ones and sparse outliers; teacher-forced against
    the oracle for 2 steps."""
    wl = W.WORKLOADS[name].replace(pool_slots=4)
    cfg = A.Config.from_workload(wl)
    mp = W.model_params(wl)
    S = _degenerate_states(wl)
    B = S.shape[0]
    slots = np.arange(B, dtype=np.int32)[::-1].copy()
    stride = A.stepq_intb_slot_bytes(cfg, bits)
    hb = O.intb_head_bytes(bits)
    pool_o = np.zeros(wl.pool_slots * stride, np.uint8)
    for b in range(B):
        for h in range(wl.hv):
            base = int(slots[b]) * stride + h * hb
            pool_o[base:base + hb] = O.intb_encode_head(S[b, h], bits)
    (slots_d,) = to_dev(slots)
    pool_d = torch.zeros(wl.pool_slots * stride, dtype=torch.uint8, device="cuda")
    t = Tally()
    for step in range(2):
        inp = W.step_inputs(wl, mp, W.STREAM_DECODE, step, 0, batch=B)
        pool_d.copy_(torch.from_numpy(pool_o))
        q, k, v, beta, gate = to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate)
        y_d = torch.empty((B, wl.hv, 128), dtype=torch.float32, device="cuda")
        A.stepq_intb_decode_step(cfg, bits, 0, pool_d, slots_d, q, k, v, beta, gate, y_d)
        y_o = O.intb_pool_step(bits, wl.hk, wl.hv, wl.gate_per_row, 0, stride, pool_o, slots, inp)
        assert np.isfinite(y_d.cpu().numpy()).all()
        compare_y(t, y_d.cpu().numpy(), y_o)
        got = pool_d.cpu().numpy()
        for b in range(B):
            for h in range(wl.hv):
                base = int(slots[b]) * stride + h * hb
                sg = got[base:base + 256].view(np.uint16)
                so = pool_o[base:base + 256].view(np.uint16)
                t.scales += 128
                t.scale_diff += int(np.count_nonzero(sg != so))
                cg = np.unpackbits(got[base + 256:base + hb], bitorder="little")
                co = np.unpackbits(pool_o[base + 256:base + hb], bitorder="little")
                ug = (cg.reshape(-1, bits) * (1 << np.arange(bits))).sum(1)
                uo = (co.reshape(-1, bits) * (1 << np.arange(bits))).sum(1)
                t.elems += ug.size
                t.code_diff += int(np.count_nonzero(ug != uo))
                t.code_maxdiff = max(t.code_maxdiff, int(np.abs(ug - uo).max()))
    # the huge slot's rows keep scales capped at FP16 65504 (0x7BFF) through the
    # step, so the clamped code path ran
    capped = got[int(slots[1]) * stride:][:256].view(np.uint16)
    assert (capped == 0x7BFF).any()
    print(bits, name, t.summary())
    t.check()
    assert A.stepq_device_error() == 0


def test_largest_head_count(torch):
    """256 value heads (64 key heads) per layer, the most one launch takes."""
    wl = W.WORKLOADS["gqa"].replace(name="maxheads", hk=64, hv=256, batch=2, pool_slots=4, n_pivots=5)
    S = W.random_states(wl, 2 * wl.hv, seed=9).reshape(2, wl.hv, 128, 128)
    t = _teacher_forced(torch, wl, S)
    print(t.summary())
    t.check()
    assert A.stepq_device_error() == 0


def test_too_many_heads_is_refused(torch):
    """More value heads than a launch supports: an error before any launch."""
    wl = W.WORKLOADS["gqa"].replace(name="toomany", hk=64, hv=320, batch=1, pool_slots=1)
    cfg, plan, oplan, _ = plans(wl, seqs=1, steps=4)
    pool_d = A.alloc_pool(plan, 1)
    before = pool_d.clone()
    z = torch.zeros((1, wl.hk, 128), device="cuda")
    zv = torch.zeros((1, wl.hv, 128), device="cuda")
    beta = torch.zeros((1, wl.hv), device="cuda")
    gate = torch.ones((1, wl.hv), device="cuda")
    slots = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(A._lib.StepqError):
        A.stepq_decode_step(plan, 0, pool_d, slots, z, z, zv, beta, gate, zv.clone())
    assert torch.equal(pool_d, before)
    assert A.stepq_device_error() == 0


@pytest.mark.parametrize("name,withhold", [("gqa", 0), ("gqa", 37), ("channel", 5)])
def test_bounded_wait_runs_out_and_recovers(torch, name, withhold):
    """Failure detection without a fault: a test switch makes the producer skip
    the copies of one item, so that item's stage barrier never completes. With
    the wait bound lowered to 1e5 cycles the kernel gives up, every CTA returns,
    and the launch reports STEPQ_ERR_TIMEOUT through the sticky error word. The
    next, normal step on the same context matches the oracle."""
    wl = W.WORKLOADS[name].replace(pool_slots=8)
    B = 4
    S = W.random_states(wl, B * wl.hv, seed=3).reshape(B, wl.hv, 128, 128)
    cfg, plan, oplan, _ = plans(wl)
    slots = np.array([6, 1, 4, 2], np.int32)
    pool_o = np.zeros(wl.pool_slots * oplan.slot_stride, np.uint8)
    O.pool_encode(oplan, pool_o, 0, slots, S)
    pool_d = torch.from_numpy(pool_o.copy()).cuda()
    inp = W.step_inputs(wl, W.model_params(wl), W.STREAM_DECODE, 0, 0, batch=B)
    q, k, v, beta, gate, slots_d = to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate, slots)
    y_d = torch.empty((B, wl.hv, 128), dtype=torch.float32, device="cuda")
    A.stepq_debug_stall(100_000, withhold)
    try:
        A.stepq_decode_step(plan, 0, pool_d, slots_d, q, k, v, beta, gate, y_d)
        assert A.stepq_device_error() == 8                                      # STEPQ_ERR_TIMEOUT
    finally:
        A.stepq_debug_stall()
    pool_d.copy_(torch.from_numpy(pool_o))
    A.stepq_decode_step(plan, 0, pool_d, slots_d, q, k, v, beta, gate, y_d)
    y_o = O.pool_step(oplan, pool_o, 0, slots, inp)
    t = Tally()
    compare_y(t, y_d.cpu().numpy(), y_o)
    compare_pools(t, pool_d.cpu().numpy(), pool_o, oplan, 0, slots)
    print(name, t.summary())
    t.check()
    assert A.stepq_device_error() == 0
