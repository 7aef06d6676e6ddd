"""Pins of the oracle's persistent decode step (App. C.3) and calibration drivers.

* Steps 1-3: the readout is taken from the updated tile before requantization
  (Eq. compressed_recurrence): it equals the FP32-state reference step applied
  to the reconstructed state; with every unit an FP16 pivot the step is exactly
  the FP32-state recurrence on FP16-rounded state.
* Prop. 1: the readout error of the compressed path is (A_t E_{t-1})^T q_t.
* Calibration (App. A.3): omega is the mean of g^2 with g = A^T q built densely.
"""
import numpy as np
import pytest

from paper_2609_38169_gb300 import workloads as W

D = 128
HEAD, ROW, PIV = 0, 1, 16


def _inp(rng, per_row):
    q = rng.standard_normal(D).astype(np.float32)
    k = rng.standard_normal(D)
    k = (k / np.linalg.norm(k)).astype(np.float32)
    v = rng.standard_normal(D).astype(np.float32)
    beta = np.float32(rng.uniform(0.1, 0.9))
    gate = (rng.uniform(0.8, 0.999, D) if per_row else [rng.uniform(0.9, 0.999)])
    return q, k, v, beta, np.asarray(gate, np.float32)


def test_pivot_head_step_is_fp32_recurrence_on_fp16_state(oracle, rng):
    S = (rng.standard_normal((D, D)) * 3).astype(np.float32)
    rb = np.full(D, PIV, np.int8)
    w = np.ones(D, np.float32)
    page = oracle.encode_head(S, HEAD, rb, w)
    S16 = oracle.decode_head_f32(page, HEAD, rb)
    assert np.array_equal(S16, np.float16(S).astype(np.float32))
    q, k, v, beta, gate = _inp(rng, False)
    page1, y = oracle.step_head(page, HEAD, rb, w, q, k, v, beta, gate)
    S1, yref = oracle.delta_step(S16, q, k, v, beta, gate)
    assert np.array_equal(y, yref)
    assert np.array_equal(oracle.decode_head_f32(page1, HEAD, rb), np.float16(S1).astype(np.float32))


@pytest.mark.parametrize("unit", [HEAD, ROW])
def test_step_reads_before_requantizing(oracle, rng, unit):
    S = (rng.standard_normal((D, D)) * np.exp(rng.normal(size=(D, 1)))).astype(np.float32)
    if unit == HEAD:
        rb = np.full(D, 6, np.int8)
    else:
        rb = rng.choice([2, 4, 6, 8], D).astype(np.int8)
        rb[:5] = PIV
    w = np.exp(rng.normal(0, 0.3, D)).astype(np.float32)
    page = oracle.encode_head(S, unit, rb, w)
    q, k, v, beta, gate = _inp(rng, unit == ROW)
    page1, y = oracle.step_head(page, unit, rb, w, q, k, v, beta, gate)
    Shat = oracle.decode_head(page, unit, rb)
    Dg = np.broadcast_to(gate.astype(np.float64), (D,))[:, None]
    k64, v64, q64 = k.astype(np.float64), v.astype(np.float64), q.astype(np.float64)
    P = Dg * Shat
    X = P + float(beta) * np.outer(k64, v64 - k64 @ P)          # Eq. delta_update, in fp64
    yref = X.T @ q64
    assert np.abs(y - yref).max() <= 2e-6 * np.abs(yref).max()
    # the new page is the fit of the fp32 tile X
    page_ref = oracle.encode_head(X.astype(np.float32), unit, rb, w)
    z1 = oracle.unpack_head(page1, unit, rb)[2]
    z2 = oracle.unpack_head(page_ref, unit, rb)[2]
    assert np.mean(z1 != z2) <= 1e-3


def test_error_propagation_prop1(oracle, rng):
    """E_t = A_t E_{t-1} + eps_t;  y_hat_t - y_t = (A_t E_{t-1})^T q_t."""
    S = (rng.standard_normal((D, D))).astype(np.float32)
    rb = np.full(D, 4, np.int8)
    w = np.ones(D, np.float32)
    page = oracle.encode_head(S, HEAD, rb, w)
    Sref = S.copy()
    for _ in range(5):
        q, k, v, beta, gate = _inp(rng, False)
        E = oracle.decode_head(page, HEAD, rb) - Sref.astype(np.float64)
        page, yq = oracle.step_head(page, HEAD, rb, w, q, k, v, beta, gate)
        Sref, yr = oracle.delta_step(Sref, q, k, v, beta, gate)
        A = (np.eye(D) - float(beta) * np.outer(k, k).astype(np.float64)) * float(gate[0])
        pred = (A @ E).T @ q.astype(np.float64)
        assert np.abs((yq.astype(np.float64) - yr) - pred).max() <= 1e-4 * np.abs(yr).max()


@pytest.mark.parametrize("name", ["gqa", "channel"])
def test_calibration_omega_and_logret(oracle, name):
    """omega sums g^2 with g = A^T q built densely; ell sums log alpha per head
    (scalar gates) or log d_i per key channel (channel gates)."""
    wl = W.WORKLOADS[name].replace(batch=3)
    mp = W.model_params(wl)
    inp = W.step_inputs(wl, mp, W.STREAM_CALIB, 0, 0, batch=3)
    grp = wl.hv // wl.hk
    om = np.zeros((wl.hv, D))
    lr = np.zeros((wl.hv, D) if wl.gate_per_row else wl.hv)
    oracle.calib_observe(inp, om, lr)
    for h in (0, 5, 31):
        ref = np.zeros(D)
        for b in range(3):
            g = oracle.row_impact(inp.q[b, h // grp], inp.k[b, h // grp], inp.beta[b, h],
                                  inp.gate[b, h], dense=True)
            ref += g * g
        assert np.allclose(om[h], ref, rtol=1e-10)
        assert np.allclose(lr[h], np.sum(np.log(inp.gate[:, h].astype(np.float64)), axis=0), rtol=1e-12)


def test_calibration_distortion_driver(oracle, rng):
    S = (rng.standard_normal((2, 3, D, D))).astype(np.float32)
    w = np.exp(rng.normal(0, 0.3, (3, D))).astype(np.float32)
    acc = np.zeros((3, 4))
    oracle.calib_distortion(HEAD, S, w, (4, 6, 8), None, 1, acc)
    for h in range(3):
        for kk, b in enumerate((4, 6, 8)):
            rb = np.full(D, b, np.int8)
            ref = 0.0
            for s in range(2):
                R = oracle.decode_head(oracle.encode_head(S[s, h], HEAD, rb, w[h]), HEAD, rb)
                ref += np.sum(w[h][:, None].astype(np.float64) ** 2 * (R - S[s, h]) ** 2) / D / D
            assert np.isclose(acc[h, kk], ref, rtol=1e-12)
        assert acc[h, 0] > acc[h, 1] > acc[h, 2] > acc[h, 3] >= 0


def test_calibration_distortion_driver_rows(oracle, rng):
    """Row units (Eq. kda_calibration_distortion): per key row, the unweighted
    mean squared error over its 128 elements, summed over the sampled states."""
    S = (rng.standard_normal((2, 2, D, D)) * np.exp(rng.normal(size=(1, 1, D, 1)))).astype(np.float32)
    w = np.exp(rng.normal(0, 0.3, (2, D))).astype(np.float32)
    cands = (2, 4, 6, 8)
    acc = np.zeros((2 * D, len(cands) + 1))
    oracle.calib_distortion(ROW, S, w, cands, None, 1, acc)
    for h in range(2):
        for kk, b in enumerate(cands):
            rb = np.full(D, b, np.int8)
            ref = np.zeros(D)
            for s in range(2):
                R = oracle.decode_head(oracle.encode_head(S[s, h], ROW, rb, w[h]), ROW, rb)
                ref += np.sum((R - S[s, h]) ** 2, axis=1) / D
            assert np.allclose(acc[h * D:(h + 1) * D, kk], ref, rtol=1e-12)
        f16 = sum(np.sum((np.float16(S[s, h]).astype(np.float64) - S[s, h]) ** 2, axis=1) / D
                  for s in range(2))
        assert np.allclose(acc[h * D:(h + 1) * D, len(cands)], f16, rtol=1e-12)


def test_end_to_end_tiny_calibration_and_plan(oracle):
    wl = W.WORKLOADS["tiny"]
    st = oracle.calibrate(wl, seqs=2, steps=32)
    plan = oracle.plan_from_stats(wl, st)
    assert plan.unit_bits.shape == (4,)
    assert np.sum(plan.unit_bits) <= 6 * 4
    assert plan.slot_stride == int(np.sum(plan.head_bytes))


@pytest.mark.parametrize("bits,per_row", [(8, False), (6, True), (4, False)])
def test_intb_step_is_recurrence_on_decoded_state(oracle, rng, bits, per_row):
    """Uniform INT-b baseline step (App. B.5): the readout is the Delta update of
    the decoded state (Eq. delta_update, fp64), and the new page is the rowwise
    encoding of that updated tile."""
    S = (rng.standard_normal((D, D)) * np.exp(rng.normal(size=(D, 1)))).astype(np.float32)
    page = oracle.intb_encode_head(S, bits)
    q, k, v, beta, gate = _inp(rng, per_row)
    page1, y = oracle.intb_step_head(page, bits, q, k, v, beta, gate)
    Shat = oracle.intb_decode_head(page, bits)
    Dg = np.broadcast_to(gate.astype(np.float64), (D,))[:, None]
    k64, v64, q64 = k.astype(np.float64), v.astype(np.float64), q.astype(np.float64)
    P = Dg * Shat
    X = P + float(beta) * np.outer(k64, v64 - k64 @ P)
    yref = X.T @ q64
    assert np.abs(y - yref).max() <= 2e-6 * np.abs(yref).max()
    ref = oracle.intb_encode_head(X.astype(np.float32), bits)
    assert np.array_equal(page1[:256], ref[:256])                     # row scales
    assert np.mean(page1[256:] != ref[256:]) <= 1e-3                   # codes (fp32 rounding ties)


def test_pool_step_is_the_per_unit_step(oracle, rng):
    """The pool driver steps each (slot, value head) unit on its own page: value
    head h reads key head h // (Hv / Hk) (grouped-query sharing), batch entry b
    works on slot slots[b], and the other slots stay untouched."""
    Hk, Hv, n_slots = 2, 4, 5
    slots = np.array([3, 0, 4], np.int32)
    B = len(slots)
    cands = (4, 6, 8)
    dist = np.sort(np.exp(rng.normal(0, 1, (Hv, 4))), axis=1)[:, ::-1].copy()
    plan = oracle.make_plan(HEAD, 1, Hk, Hv, 6, cands, 1, 64, 1,
                            np.exp(rng.normal(0, 1, (1, Hv, D))).astype(np.float32),
                            rng.normal(-0.02, 0.01, Hv), dist)
    pool = np.zeros(n_slots * plan.slot_stride, np.uint8)
    states = rng.standard_normal((B, Hv, D, D)).astype(np.float32)
    oracle.pool_encode(plan, pool, 0, slots, states)
    before = pool.copy()

    class Inp:
        pass
    inp = Inp()
    inp.q = rng.standard_normal((B, Hk, D)).astype(np.float32)
    inp.k = rng.standard_normal((B, Hk, D)).astype(np.float32)
    inp.k /= np.linalg.norm(inp.k, axis=-1, keepdims=True)
    inp.v = rng.standard_normal((B, Hv, D)).astype(np.float32)
    inp.beta = rng.uniform(0.1, 0.9, (B, Hv)).astype(np.float32)
    inp.gate = rng.uniform(0.9, 0.999, (B, Hv)).astype(np.float32)
    y = oracle.pool_step(plan, pool, 0, slots, inp)
    rb_layer, w_layer = plan.layer_row_bits(0), plan.layer_w(0)
    for b in range(B):
        for h in range(Hv):
            o = int(slots[b]) * plan.slot_stride + int(plan.head_off[h])
            n = int(plan.head_bytes[h])
            page1, yu = oracle.step_head(before[o:o + n], HEAD, rb_layer[h], w_layer[h],
                                         inp.q[b, h // 2], inp.k[b, h // 2], inp.v[b, h],
                                         inp.beta[b, h], inp.gate[b, h])
            assert np.array_equal(y[b, h], yu)
            assert np.array_equal(pool[o:o + n], page1)
    for s in set(range(n_slots)) - set(slots.tolist()):
        seg = slice(s * plan.slot_stride, (s + 1) * plan.slot_stride)
        assert np.array_equal(pool[seg], before[seg])


@pytest.mark.parametrize("gate_kind", ["scalar", "channel"])
def test_reported_residual_matches_the_readout(oracle, rng, gate_kind):
    """The residual delta = v - k^T D S_hat that the step reports (App. C.3 step 2)
    is the one its update applied: with X = D S_hat + beta k delta^T, the readout
    satisfies y - (D S_hat)^T q = beta (q . k) delta (Eq. compressed_recurrence),
    up to the fp32 rounding of X."""
    Hk, Hv, n_slots = 2, 4, 3
    slots = np.array([2, 0], np.int32)
    B = len(slots)
    unit = HEAD if gate_kind == "scalar" else ROW
    cands = (4, 6, 8)
    units = Hv if unit == HEAD else Hv * D
    dist = np.sort(np.exp(rng.normal(0, 1, (units, 4))), axis=1)[:, ::-1].copy()
    plan = oracle.make_plan(unit, 1, Hk, Hv, 6, cands, 0, 64, 1,
                            np.exp(rng.normal(0, 1, (1, Hv, D))).astype(np.float32),
                            rng.normal(-0.02, 0.01, units), dist)
    pool = np.zeros(n_slots * plan.slot_stride, np.uint8)
    oracle.pool_encode(plan, pool, 0, slots, rng.standard_normal((B, Hv, D, D)).astype(np.float32))
    S_hat = oracle.pool_decode(plan, pool, 0, slots).astype(np.float64)

    class Inp:
        pass
    inp = Inp()
    inp.q = rng.standard_normal((B, Hk, D)).astype(np.float32)
    inp.k = rng.standard_normal((B, Hk, D)).astype(np.float32)
    inp.k /= np.linalg.norm(inp.k, axis=-1, keepdims=True)
    inp.v = rng.standard_normal((B, Hv, D)).astype(np.float32)
    inp.beta = rng.uniform(0.1, 0.9, (B, Hv)).astype(np.float32)
    gshape = (B, Hv) if unit == HEAD else (B, Hv, D)
    inp.gate = rng.uniform(0.9, 0.999, gshape).astype(np.float32)
    y, delta = oracle.pool_step(plan, pool, 0, slots, inp, with_delta=True)
    q = np.repeat(inp.q.astype(np.float64), Hv // Hk, axis=1)
    k = np.repeat(inp.k.astype(np.float64), Hv // Hk, axis=1)
    g = inp.gate.astype(np.float64)
    g = g[..., None, None] if unit == HEAD else g[..., :, None]
    base = np.einsum("bhi,bhij->bhj", q, g * S_hat)
    lhs = y.astype(np.float64) - base
    rhs = inp.beta.astype(np.float64)[..., None] * np.einsum("bhi,bhi->bh", q, k)[..., None] * delta
    scale = np.einsum("bhi,bhij->bhj", np.abs(q), np.abs(g * S_hat)).max(axis=-1, keepdims=True)
    assert np.all(np.abs(lhs - rhs) <= 1e-5 * scale)
    assert np.abs(rhs).max() > 1e-3 * np.abs(lhs).max()       # the term is not negligible
