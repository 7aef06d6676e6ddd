"""The decode step split for a side stream (Sec. 4.4, App. F.1): the readout
returns y and delta and leaves the pages as they are; the writeback refits and
packs (App. C.3 steps 6-7: the old representation stays valid until its
readers are done).

Both halves are checked against the oracle under the parity rules of
gpu_helpers, teacher-forced: y and the written pages against the oracle's
decode step from the same packed pool, delta against the oracle's retrieval
residual v - k^T D S_hat. As a property of the split, the readout must also
return the fused step's y bit for bit and the writeback write its pages byte
for byte, also when the two halves run on different CUDA streams over several
steps."""
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


def _setup(torch, name, kw, B, layer):
    wl = W.WORKLOADS[name].replace(**kw)
    cfg, plan, oplan, _ = plans(wl)
    slots = np.random.default_rng(3).permutation(wl.pool_slots)[:B].astype(np.int32)
    pool_o = np.zeros(wl.pool_slots * oplan.slot_stride, np.uint8)
    O.pool_encode(oplan, pool_o, layer, slots, O.warmup_states(wl, layer, B))
    return wl, plan, oplan, slots, pool_o


def _compare_delta(delta_gpu, delta_ora, inp, S_hat, wl):
    """delta is fp32 on the GPU: each element within 1e-5 of the magnitudes that
    enter it, |v_j| + max_i |k_i (D S_hat)_ij| (the retrieval's fp32 sum)."""
    grp = wl.hv // wl.hk
    kk = np.repeat(inp.k.astype(np.float64), grp, axis=1)
    g = inp.gate.astype(np.float64)
    g = g if g.ndim == 3 else g[..., None]
    u_abs = np.abs(np.einsum("bhi,bhij->bhj", np.abs(kk * g), np.abs(S_hat)))
    scale = np.abs(inp.v).max(axis=-1) + u_abs.max(axis=-1)
    err = np.abs(delta_gpu.astype(np.float64) - delta_ora).max(axis=-1)
    assert (err <= 1e-5 * scale).all(), (err / scale).max()


@pytest.mark.parametrize("name,kw,layer", [("gqa", dict(n_pivots=3), 0),
                                           ("pool", dict(layers=2, pool_slots=64, batch=16), 1),
                                           ("channel", {}, 0),
                                           ("drift", dict(layers=2, pool_slots=32, batch=16), 1),
                                          ("gqa", dict(nominal_bits=4, candidates=(2, 4, 6, 8), n_pivots=2), 0)])
def test_readout_and_writeback_against_the_oracle(torch, name, kw, layer):
    B = 16
    wl, plan, oplan, slots, pool_o = _setup(torch, name, kw, B, layer)
    assert (oplan.unit_bits == 16).any()
    inp = W.step_inputs(wl, W.model_params(wl), W.STREAM_DECODE, 0, layer, batch=B)
    S_hat = O.pool_decode(oplan, pool_o, layer, slots).astype(np.float64)
    q, k, v, beta, gate, slots_d = to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate, slots)
    (pool0,) = to_dev(pool_o)
    pool_f, pool_s = pool0.clone(), pool0.clone()
    y_f = torch.empty((B, wl.hv, 128), dtype=torch.float32, device="cuda")
    y_r, delta = torch.empty_like(y_f), torch.empty_like(y_f)
    A.stepq_decode_readout(plan, layer, pool_s, slots_d, q, k, v, beta, gate, y_r, delta)
    torch.cuda.synchronize()
    assert torch.equal(pool_s, pool0)                      # the readout writes no page
    A.stepq_decode_writeback(plan, layer, pool_s, slots_d, k, beta, gate, delta)
    pool_new = pool_o.copy()
    y_o, d_o = O.pool_step(oplan, pool_new, layer, slots, inp, with_delta=True)
    t = Tally()
    compare_y(t, y_r.cpu().numpy(), y_o)
    compare_pools(t, pool_s.cpu().numpy(), pool_new, oplan, layer, slots)
    print(name, t.summary())
    t.check()
    _compare_delta(delta.cpu().numpy(), d_o, inp, S_hat, wl)
    # the split against the fused step
    A.stepq_decode_step(plan, layer, pool_f, slots_d, q, k, v, beta, gate, y_f)
    assert torch.equal(y_r, y_f)
    assert torch.equal(pool_s, pool_f)
    assert A.stepq_device_error() == 0


@pytest.mark.parametrize("name,kw", [("gqa", dict(n_pivots=3)), ("channel", {})])
def test_split_on_two_streams_over_steps(torch, name, kw):
    """Readout on the main stream, writeback on a side stream ordered by events,
    for 4 steps. Teacher-forced against the oracle: each step starts both sides
    from the oracle's pool of the previous step. Free-running, the split matches
    4 fused steps bit for bit."""
    B, layer, steps = 16, 0, 4
    wl, plan, oplan, slots, pool_o = _setup(torch, name, kw, B, layer)
    mp = W.model_params(wl)
    (pool0, slots_d) = to_dev(pool_o, slots)
    main, side = torch.cuda.Stream(), torch.cuda.Stream()
    inps = [W.step_inputs(wl, mp, W.STREAM_DECODE, t, layer, batch=B) for t in range(steps)]
    inputs = [to_dev(i.q, i.k, i.v, i.beta, i.gate) for i in inps]
    torch.cuda.synchronize()

    def split_step(pool, t, y, d, done):
        q, k, v, beta, gate = inputs[t]
        with torch.cuda.stream(main):
            if done is not None:
                main.wait_event(done)                      # writeback before the next read
            A.stepq_decode_readout(plan, layer, pool, slots_d, q, k, v, beta, gate, y, d, stream=main)
            ready = torch.cuda.Event()
            ready.record(main)
        with torch.cuda.stream(side):
            side.wait_event(ready)
            A.stepq_decode_writeback(plan, layer, pool, slots_d, k, beta, gate, d, stream=side)
            done = torch.cuda.Event()
            done.record(side)
        return done

    # teacher-forced against the oracle
    tally = Tally()
    pool_t = pool0.clone()
    y_t = torch.empty((B, wl.hv, 128), dtype=torch.float32, device="cuda")
    d_t = torch.empty_like(y_t)
    ora = pool_o.copy()
    for t in range(steps):
        pool_t.copy_(torch.from_numpy(ora))
        torch.cuda.synchronize()
        split_step(pool_t, t, y_t, d_t, None)
        torch.cuda.synchronize()
        y_o = O.pool_step(oplan, ora, layer, slots, inps[t])
        compare_y(tally, y_t.cpu().numpy(), y_o)
        compare_pools(tally, pool_t.cpu().numpy(), ora, oplan, layer, slots)
    print(name, tally.summary())
    tally.check()

    # free-running: the split equals the fused step
    pool_f, pool_s = pool0.clone(), pool0.clone()
    y_f = torch.empty((steps, B, wl.hv, 128), dtype=torch.float32, device="cuda")
    y_s, delta = torch.empty_like(y_f), torch.empty_like(y_f)
    for t, (q, k, v, beta, gate) in enumerate(inputs):
        A.stepq_decode_step(plan, layer, pool_f, slots_d, q, k, v, beta, gate, y_f[t])
    done = None
    for t in range(steps):
        done = split_step(pool_s, t, y_s[t], delta[t], done)
    torch.cuda.synchronize()
    assert torch.equal(y_s, y_f)
    assert torch.equal(pool_s, pool_f)
    assert A.stepq_device_error() == 0
