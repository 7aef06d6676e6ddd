"""GPU parity of the CUDA path against the CPU oracle, through the C ABI.

Every case feeds both sides the same seeded inputs; the oracle's results are
never computed from the GPU's. Decode steps are teacher-forced: each step starts
both sides from the oracle's packed pool of the previous step.
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


def _slots(wl, batch, seed=11):
    g = np.random.default_rng(seed)
    return g.permutation(wl.pool_slots)[:batch].astype(np.int32)


@pytest.mark.parametrize("name,kw,batch", [
    ("tiny", {}, 1),
    ("gqa", {}, 64),
    ("channel", {}, 24),
    ("gqa", dict(n_pivots=3), 8),
    ("channel", dict(nominal_bits=6, candidates=(4, 6, 8), n_pivots=40), 8),
    ("gqa", dict(nominal_bits=4, candidates=(2, 4, 6, 8), n_pivots=2), 16),    # 2-bit heads
])
def test_quantize_dequantize_pool(torch, name, kw, batch):
    """Pack fp32 states (App. C.3 steps 4-6) and unpack them again."""
    wl = W.WORKLOADS[name].replace(**kw)
    cfg, plan, oplan, _ = plans(wl)
    slots = _slots(wl, batch)
    S = W.random_states(wl, batch * wl.hv).reshape(batch, wl.hv, 128, 128)
    pool_o = np.zeros(wl.pool_slots * oplan.slot_stride, np.uint8)
    O.pool_encode(oplan, pool_o, 0, slots, S)
    S_d, slots_d = to_dev(S, slots)
    pool_d = A.alloc_pool(plan, wl.pool_slots)
    A.stepq_quantize_pool(plan, 0, S_d, slots_d, pool_d)
    t = Tally()
    compare_pools(t, pool_d.cpu().numpy(), pool_o, oplan, 0, slots)
    t.y_worst = 0.0
    t.check()
    # dequantize the oracle's pool: bit-exact reconstruction r_i c_j z_ij
    pool_d.copy_(torch.from_numpy(pool_o))
    out = torch.empty_like(S_d)
    A.stepq_dequantize_pool(plan, 0, pool_d, slots_d, out)
    ref = O.pool_decode(oplan, pool_o, 0, slots)
    assert np.array_equal(out.cpu().numpy(), ref)
    assert A.stepq_device_error() == 0


@pytest.mark.parametrize("name,kw,batch,steps", [
    ("tiny", {}, 1, 64),
    ("gqa", {}, 64, 6),
    ("channel", {}, 32, 6),
    ("gqa", dict(n_pivots=3), 16, 4),
    ("channel", dict(nominal_bits=6, candidates=(4, 6, 8), n_pivots=40), 16, 4),
    ("tiny", dict(fit_iters=3), 1, 8),
    ("gqa", dict(nominal_bits=4, candidates=(2, 4, 6, 8), n_pivots=2), 16, 4),  # 2-bit heads
    ("channel", dict(fit_iters=2), 16, 3),                                     # row units, two LS passes
    ("gqa", dict(fit_iters=2), 16, 3),                                         # head units, two LS passes
])
def test_decode_step_teacher_forced(torch, name, kw, batch, steps):
    """App. C.3 steps 1-7 against the oracle, step by step."""
    wl = W.WORKLOADS[name].replace(**kw)
    cfg, plan, oplan, _ = plans(wl)
    mp = W.model_params(wl)
    slots = _slots(wl, batch)
    S0 = O.warmup_states(wl, 0, batch)
    pool_o = np.zeros(wl.pool_slots * oplan.slot_stride, np.uint8)
    O.pool_encode(oplan, pool_o, 0, slots, S0)
    (slots_d,) = to_dev(slots)
    pool_d = A.alloc_pool(plan, wl.pool_slots)
    t = Tally()
    for step in range(steps):
        inp = W.step_inputs(wl, mp, W.STREAM_DECODE, step, 0, batch=batch)
        pool_d.copy_(torch.from_numpy(pool_o))
        q, k, v, beta, gate = to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate)
        y_d = torch.empty((batch, wl.hv, 128), dtype=torch.float32, device="cuda")
        A.stepq_decode_step(plan, 0, pool_d, slots_d, q, k, v, beta, gate, y_d)
        y_o = O.pool_step(oplan, pool_o, 0, slots, inp)
        compare_y(t, y_d.cpu().numpy(), y_o)
        compare_pools(t, pool_d.cpu().numpy(), pool_o, oplan, 0, slots)
    print(name, kw, t.summary())
    t.check()
    assert A.stepq_device_error() == 0


def test_fp32_state_decode(torch):
    """FP32-state baseline = Eq. delta_update with the state kept in fp32."""
    wl = W.WORKLOADS["gqa"]
    cfg = A.Config.from_workload(wl)
    mp = W.model_params(wl)
    B = 16
    slots = _slots(wl, B)
    S = W.random_states(wl, B * wl.hv).reshape(B, wl.hv, 128, 128)
    pool = np.zeros((wl.pool_slots, 1, wl.hv, 128, 128), np.float32)
    pool[slots, 0] = S
    (pool_d, slots_d) = to_dev(pool, slots)
    inp = W.step_inputs(wl, mp, W.STREAM_DECODE, 0, 0, batch=B)
    q, k, v, beta, gate = to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate)
    y_d = torch.empty((B, wl.hv, 128), dtype=torch.float32, device="cuda")
    A.stepq_fp32_decode_step(cfg, 0, pool_d, slots_d, q, k, v, beta, gate, y_d)
    S_o = S.copy()
    y_o = O.delta_batch(S_o, inp.q, inp.k, inp.v, inp.beta, inp.gate)
    t = Tally()
    compare_y(t, y_d.cpu().numpy(), y_o)
    assert t.y_worst <= 1e-5
    got = pool_d.cpu().numpy()[slots, 0]
    assert np.abs(got - S_o).max() <= 1e-5 * np.abs(S_o).max()


@pytest.mark.parametrize("name", ["gqa", "channel"])
def test_fp32_exact_read_decode(torch, name):
    """Exact-read step of the feedback experiment (App. B.1): the residual reads
    a separate reference pool, which the kernel leaves untouched."""
    wl = W.WORKLOADS[name]
    cfg = A.Config.from_workload(wl)
    mp = W.model_params(wl)
    B = 12
    slots = _slots(wl, B)
    S_ref = W.random_states(wl, B * wl.hv).reshape(B, wl.hv, 128, 128)
    rng = np.random.default_rng(11)
    S = (S_ref + 0.05 * np.abs(S_ref).max() * rng.standard_normal(S_ref.shape)).astype(np.float32)
    pool = np.zeros((wl.pool_slots, 1, wl.hv, 128, 128), np.float32)
    rpool = np.zeros_like(pool)
    pool[slots, 0] = S
    rpool[slots, 0] = S_ref
    (pool_d, rpool_d, slots_d) = to_dev(pool, rpool, slots)
    inp = W.step_inputs(wl, mp, W.STREAM_DECODE, 3, 0, batch=B)
    q, k, v, beta, gate = to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate)
    y_d = torch.empty((B, wl.hv, 128), dtype=torch.float32, device="cuda")
    A.stepq_fp32_exact_read_step(cfg, 0, pool_d, rpool_d, slots_d, q, k, v, beta, gate, y_d)
    S_o = S.copy()
    y_o = O.delta_batch_read(S_o, S_ref, inp.q, inp.k, inp.v, inp.beta, inp.gate)
    t = Tally()
    compare_y(t, y_d.cpu().numpy(), y_o)
    assert t.y_worst <= 1e-5
    got = pool_d.cpu().numpy()[slots, 0]
    assert np.abs(got - S_o).max() <= 1e-5 * np.abs(S_o).max()
    assert np.array_equal(rpool_d.cpu().numpy(), rpool)
    assert A.stepq_device_error() == 0


@pytest.mark.parametrize("name,kw", [("gqa", dict(n_pivots=3)), ("channel", {})])
def test_temporal_codec(torch, name, kw):
    """"Temporal only" ablation codec (Sec. 5.4): the plan's widths and FP16
    pivots with the rowwise quantizer of App. B.5; pack is byte-exact against the
    oracle and unpack reproduces the oracle's decode exactly."""
    wl = W.WORKLOADS[name].replace(**kw)
    cfg, plan, oplan, _ = plans(wl)
    B = 8
    slots = _slots(wl, B)
    stride = A.stepq_temporal_slot_bytes(plan)
    rb = oplan.layer_row_bits(0)
    hb = [O.temporal_head_bytes(rb[h]) for h in range(wl.hv)]
    off = np.concatenate([[0], np.cumsum(hb)])
    S = W.random_states(wl, B * wl.hv).reshape(B, wl.hv, 128, 128)
    pool_o = np.zeros(wl.pool_slots * stride, np.uint8)
    ref = np.zeros_like(S)
    for b in range(B):
        for h in range(wl.hv):
            base = int(slots[b]) * stride + int(off[h])
            pool_o[base:base + hb[h]] = O.temporal_encode_head(S[b, h], rb[h])
            ref[b, h] = O.temporal_decode_head(pool_o[base:base + hb[h]], rb[h])
    assert (rb == 16).any()
    S_d, slots_d = to_dev(S, slots)
    pool_d = torch.zeros(wl.pool_slots * stride, dtype=torch.uint8, device="cuda")
    A.stepq_temporal_quantize_pool(plan, 0, S_d, slots_d, pool_d)
    assert np.array_equal(pool_d.cpu().numpy(), pool_o)
    out = torch.empty_like(S_d)
    A.stepq_temporal_dequantize_pool(plan, 0, pool_d, slots_d, out)
    assert np.array_equal(out.cpu().numpy(), ref)
    assert A.stepq_device_error() == 0


@pytest.mark.parametrize("bits,name", [(8, "gqa"), (4, "channel"), (6, "gqa"), (6, "channel")])
def test_intb_decode(torch, bits, name):
    """Uniform rowwise-absmax INT-b state (App. B.5), teacher-forced for 3 steps."""
    wl = W.WORKLOADS[name]
    cfg = A.Config.from_workload(wl)
    mp = W.model_params(wl)
    B = 8
    slots = _slots(wl, B)
    stride = A.stepq_intb_slot_bytes(cfg, bits)
    hb = O.intb_head_bytes(bits)
    S = W.random_states(wl, B * wl.hv).reshape(B, wl.hv, 128, 128)
    pool_o = np.zeros(wl.pool_slots * stride, np.uint8)
    for b in range(B):
        for h in range(wl.hv):
            base = int(slots[b]) * stride + h * hb
            pool_o[base:base + hb] = O.intb_encode_head(S[b, h], bits)
    S_d, slots_d = to_dev(S, slots)
    pool_d = torch.zeros(wl.pool_slots * stride, dtype=torch.uint8, device="cuda")
    A.stepq_intb_quantize_pool(cfg, bits, 0, S_d, slots_d, pool_d)
    assert np.array_equal(pool_d.cpu().numpy(), pool_o)
    out = torch.empty_like(S_d)
    A.stepq_intb_dequantize_pool(cfg, bits, 0, pool_d, slots_d, out)
    ref = np.stack([np.stack([O.intb_decode_head(pool_o[int(slots[b]) * stride + h * hb:][:hb], bits)
                              for h in range(wl.hv)]) for b in range(B)])
    assert np.array_equal(out.cpu().numpy(), ref.astype(np.float32))
    t = Tally()
    for step in range(3):
        inp = W.step_inputs(wl, mp, W.STREAM_DECODE, step, 0, batch=B)
        pool_d.copy_(torch.from_numpy(pool_o))
        q, k, v, beta, gate = to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate)
        y_d = torch.empty((B, wl.hv, 128), dtype=torch.float32, device="cuda")
        A.stepq_intb_decode_step(cfg, bits, 0, pool_d, slots_d, q, k, v, beta, gate, y_d)
        y_o = O.intb_pool_step(bits, wl.hk, wl.hv, wl.gate_per_row, 0, stride, pool_o, slots, inp)
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
    print(bits, name, t.summary())
    t.check()


@pytest.mark.parametrize("name", ["tiny", "channel"])
def test_calibration_statistics(torch, name):
    """Device calibration (App. A.3) against the oracle's on the same stream."""
    wl = W.WORKLOADS[name].replace(layers=1)
    cfg = A.Config.from_workload(wl)
    st_o = O.calibrate(wl, seqs=2, steps=16)
    st_g = A.calibrate(cfg, wl, seqs=2, steps=16)
    assert np.allclose(st_g.omega, st_o.omega, rtol=1e-5)
    assert np.allclose(st_g.mean_log_ret, st_o.mean_log_ret, rtol=1e-9, atol=1e-12)
    assert np.allclose(st_g.dist_stage1, st_o.dist_stage1, rtol=2e-3)
    assert np.allclose(st_g.dist, st_o.dist, rtol=2e-3)


def test_empty_batch_and_bad_slots(torch):
    wl = W.WORKLOADS["tiny"]
    cfg, plan, oplan, _ = plans(wl)
    pool_d = A.alloc_pool(plan, 4)
    before = pool_d.clone()
    q = torch.zeros((1, 4, 128), device="cuda")
    v = torch.zeros((1, 4, 128), device="cuda")
    beta = torch.zeros((1, 4), device="cuda")
    gate = torch.ones((1, 4), device="cuda")
    y = torch.zeros((1, 4, 128), device="cuda")
    empty = torch.zeros(0, dtype=torch.int32, device="cuda")
    A.stepq_decode_step(plan, 0, pool_d, empty, q, q, v, beta, gate, y)         # B = 0: no-op
    bad = torch.tensor([7], dtype=torch.int32, device="cuda")                  # >= pool_slots
    A.stepq_decode_step(plan, 0, pool_d, bad, q, q, v, beta, gate, y, pool_slots=4)
    assert A.stepq_device_error() == 2                                          # STEPQ_ERR_SLOT_RANGE
    assert A.stepq_device_error() == 0                                          # cleared
    A.stepq_decode_step(plan, 0, pool_d, bad, q, q, v, beta, gate, y, pool_slots=4)
    assert A.stepq_stream_status() == 2                                         # same word, other name
    assert A.stepq_stream_status() == 0
    assert torch.equal(pool_d, before)
    with pytest.raises(A._lib.StepqError):
        A.stepq_decode_step(plan, 1, pool_d, bad, q, q, v, beta, gate, y)       # layer out of range
    scratch = torch.zeros(1, dtype=torch.int32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    dup = torch.tensor([0, 2, 0], dtype=torch.int32, device="cuda")
    A.stepq_validate_slots(dup, 4, scratch, status)
    assert int(status.item()) == 3
    A.stepq_validate_slots(torch.tensor([3, 1], dtype=torch.int32, device="cuda"), 4, scratch, status)
    assert int(status.item()) == 0


@pytest.mark.parametrize("kind", ["heads", "heads_readout", "heads_writeback", "rows", "fp32", "int8"])
@pytest.mark.parametrize("slots_list", [[1, 3, 1], [5, 0, 2, 4, 6, 7, 9, 5]])
def test_repeated_slots_are_reported(torch, kind, slots_list):
    """A slot id repeated within one call (two units writing one page) raises
    STEPQ_ERR_DUP_SLOT on the device; a call with distinct ids raises nothing.
    The second list repeats its first entry at the last position (the pair
    enumeration's wrap-around)."""
    wl = W.WORKLOADS["channel" if kind == "rows" else "tiny"].replace(pool_slots=16)
    cfg, plan, oplan, _ = plans(wl)
    B = len(slots_list)
    hk, hv = wl.hk, wl.hv
    gshape = (B, hv, 128) if wl.gate_per_row else (B, hv)
    q = torch.randn((B, hk, 128), device="cuda")
    k = torch.nn.functional.normalize(torch.randn((B, hk, 128), device="cuda"), dim=-1)
    v = torch.randn((B, hv, 128), device="cuda")
    beta = torch.full((B, hv), 0.5, device="cuda")
    gate = torch.full(gshape, 0.95, device="cuda")
    y = torch.empty((B, hv, 128), device="cuda")
    delta = torch.zeros((B, hv, 128), device="cuda")
    if kind == "fp32":
        pool = torch.zeros((wl.pool_slots, wl.layers, hv, 128, 128), device="cuda")
    elif kind == "int8":
        pool = torch.zeros(wl.pool_slots * A.stepq_intb_slot_bytes(cfg, 8), dtype=torch.uint8, device="cuda")
    else:
        pool = A.alloc_pool(plan, wl.pool_slots)

    def call(sl):
        s_d = torch.tensor(sl, dtype=torch.int32, device="cuda")
        if kind in ("heads", "rows"):
            A.stepq_decode_step(plan, 0, pool, s_d, q, k, v, beta, gate, y)
        elif kind == "heads_readout":
            A.stepq_decode_readout(plan, 0, pool, s_d, q, k, v, beta, gate, y, delta)
        elif kind == "heads_writeback":
            A.stepq_decode_writeback(plan, 0, pool, s_d, k, beta, gate, delta)
        elif kind == "fp32":
            A.stepq_fp32_decode_step(cfg, 0, pool, s_d, q, k, v, beta, gate, y)
        else:
            A.stepq_intb_decode_step(cfg, 8, 0, pool, s_d, q, k, v, beta, gate, y)

    call(slots_list)
    assert A.stepq_device_error() == 3                                          # STEPQ_ERR_DUP_SLOT
    call(list(range(B)))
    assert A.stepq_device_error() == 0
