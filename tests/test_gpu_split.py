"""The decode step split for a side stream (Sec. 4.4, App. F.1): the readout
returns y and delta and leaves the pages as they are; the writeback refits and
packs. Together they reproduce the fused step exactly: y bit for bit and the
pages byte for byte, also when the two halves run on different CUDA streams
over several steps."""
import numpy as np
import pytest

import oracle as O
from paper_2609_38169_gb300 import api as A, workloads as W

from gpu_helpers import plans, to_dev

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


@pytest.mark.parametrize("name,kw,layer", [("gqa", dict(n_pivots=3), 0),
                                           ("pool", dict(layers=2, pool_slots=64, batch=16), 1),
                                           ("channel", {}, 0),
                                           ("drift", dict(layers=2, pool_slots=32, batch=16), 1),
                                          ("gqa", dict(nominal_bits=4, candidates=(2, 4, 6, 8), n_pivots=2), 0)])
def test_readout_then_writeback_is_the_fused_step(torch, name, kw, layer):
    B = 16
    wl, plan, oplan, slots, pool_o = _setup(torch, name, kw, B, layer)
    assert (oplan.unit_bits == 16).any()
    inp = W.step_inputs(wl, W.model_params(wl), W.STREAM_DECODE, 0, layer, batch=B)
    q, k, v, beta, gate, slots_d = to_dev(inp.q, inp.k, inp.v, inp.beta, inp.gate, slots)
    (pool0,) = to_dev(pool_o)
    pool_f, pool_s = pool0.clone(), pool0.clone()
    y_f = torch.empty((B, wl.hv, 128), dtype=torch.float32, device="cuda")
    y_r, delta = torch.empty_like(y_f), torch.empty_like(y_f)
    A.stepq_decode_step(plan, layer, pool_f, slots_d, q, k, v, beta, gate, y_f)
    A.stepq_decode_readout(plan, layer, pool_s, slots_d, q, k, v, beta, gate, y_r, delta)
    torch.cuda.synchronize()
    assert torch.equal(pool_s, pool0)                      # the readout writes no page
    assert torch.equal(y_r, y_f)
    A.stepq_decode_writeback(plan, layer, pool_s, slots_d, k, beta, gate, delta)
    assert torch.equal(pool_s, pool_f)
    # delta_j = v_j - sum_i k_i d_i S_hat_ij with S_hat the oracle's decode of the old pages
    S_hat = O.pool_decode(oplan, pool_o, layer, slots).astype(np.float64)
    grp = wl.hv // wl.hk
    kk = np.repeat(inp.k.astype(np.float64), grp, axis=1)
    g = inp.gate.astype(np.float64)
    g = g if g.ndim == 3 else g[..., None]                 # per key channel or per head
    u = np.einsum("bhi,bhij->bhj", kk * g, S_hat)
    d_o = inp.v - u
    err = np.abs(delta.cpu().numpy() - d_o).max(axis=-1)
    scale = np.abs(inp.v).max(axis=-1) + np.abs(u).max(axis=-1)
    assert (err <= 1e-5 * scale).all(), (err / scale).max()
    assert A.stepq_device_error() == 0


@pytest.mark.parametrize("name,kw", [("gqa", dict(n_pivots=3)), ("channel", {})])
def test_split_on_two_streams_over_steps(torch, name, kw):
    """Readout on the main stream, writeback on a side stream ordered by events,
    for 4 steps: the same pages and outputs as 4 fused steps."""
    B, layer, steps = 16, 0, 4
    wl, plan, oplan, slots, pool_o = _setup(torch, name, kw, B, layer)
    mp = W.model_params(wl)
    (pool0, slots_d) = to_dev(pool_o, slots)
    pool_f, pool_s = pool0.clone(), pool0.clone()
    main, side = torch.cuda.Stream(), torch.cuda.Stream()
    y_f = torch.empty((steps, B, wl.hv, 128), dtype=torch.float32, device="cuda")
    y_s, delta = torch.empty_like(y_f), torch.empty_like(y_f)
    inputs = [to_dev(*(lambda i: (i.q, i.k, i.v, i.beta, i.gate))(
        W.step_inputs(wl, mp, W.STREAM_DECODE, t, layer, batch=B))) for t in range(steps)]
    torch.cuda.synchronize()
    for t, (q, k, v, beta, gate) in enumerate(inputs):
        A.stepq_decode_step(plan, layer, pool_f, slots_d, q, k, v, beta, gate, y_f[t])
    done = None
    for t, (q, k, v, beta, gate) in enumerate(inputs):
        with torch.cuda.stream(main):
            if done is not None:
                main.wait_event(done)                      # writeback before the next read
            A.stepq_decode_readout(plan, layer, pool_s, slots_d, q, k, v, beta, gate, y_s[t],
                                   delta[t], stream=main)
            ready = torch.cuda.Event()
            ready.record(main)
        with torch.cuda.stream(side):
            side.wait_event(ready)
            A.stepq_decode_writeback(plan, layer, pool_s, slots_d, k, beta, gate, delta[t],
                                     stream=side)
            done = torch.cuda.Event()
            done.record(side)
    torch.cuda.synchronize()
    assert torch.equal(y_s, y_f)
    assert torch.equal(pool_s, pool_f)
    assert A.stepq_device_error() == 0
