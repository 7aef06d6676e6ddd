"""Full-size parity in the launch configuration of each workload's timing: every
active slot of the pool in a random permutation, one launch per layer-step.

- the 1024-slot serving pool (16 layers x 32 heads, head units, the bench's
  workload);
- the channel-gate decode workload (1 layer x 32 heads, 256 slots, row units
  at 4 bits);
- the drift workload's pool (4 layers x 32 heads, 128 slots, row units at 6
  bits).

The whole pool is packed on the GPU; a sample of (slot, layer, head) units gets
pages packed by the oracle from its own states instead, so the oracle can step
exactly those units one by one and compare outputs and pages.
"""
import numpy as np
import pytest

import oracle as O
from paper_2609_38169_gb300 import api as A, workloads as W

from gpu_helpers import Tally, compare_head, compare_y

pytestmark = pytest.mark.gpu


def _sample_heads(oplan, layer, Hv, rng):
    """Every FP16 pivot head and one head per width (head units), or the heads
    holding pivot rows (row units, at most four), plus six random heads."""
    if oplan.unit_kind == O.UNIT_HEAD:
        bits = oplan.unit_bits[layer * Hv:(layer + 1) * Hv]
        heads = list(np.flatnonzero(bits == 16)) + [int(np.flatnonzero(bits == b)[0])
                                                    for b in (2, 4, 6, 8) if np.any(bits == b)]
    else:
        rows = oplan.unit_bits.reshape(oplan.n_layers, Hv, 128)[layer]
        heads = list(np.flatnonzero((rows == 16).any(axis=1))[:4])
    return [int(h) for h in heads] + [int(h) for h in rng.choice(Hv, 6, replace=False)]


@pytest.mark.parametrize("name,layers", [("pool", [0, 7, 15]), ("channel", [0]), ("drift", [0, 3])])
def test_full_size_sampled(name, layers):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    wl = W.WORKLOADS[name]
    st = O.calibrate(wl, seqs=2, steps=8)
    oplan = O.plan_from_stats(wl, st)
    cfg = A.Config.from_workload(wl)
    plan = A.stepq_fit_scales(cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
    assert np.array_equal(plan.unit_bits, oplan.unit_bits)
    assert plan.slot_stride == oplan.slot_stride
    dev = torch.device("cuda", 0)
    L, Hv, Hk, B = wl.layers, wl.hv, wl.hk, wl.batch
    pool = A.alloc_pool(plan, wl.pool_slots, dev)
    all_slots = torch.arange(wl.pool_slots, dtype=torch.int32, device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(1234)
    for layer in range(L):
        S = torch.randn((wl.pool_slots, Hv, 128, 128), generator=g, device=dev)
        S *= torch.exp(torch.randn((wl.pool_slots, Hv, 128, 1), generator=g, device=dev))
        A.stepq_quantize_pool(plan, layer, S, all_slots, pool)
        del S
    torch.cuda.synchronize()
    slots = W.slot_permutation(wl)
    slots_d = torch.from_numpy(slots).to(dev)

    rng = np.random.default_rng(7)
    units = {}
    for layer in layers:
        heads = _sample_heads(oplan, layer, Hv, rng)
        units[layer] = [(int(rng.integers(B)), h) for h in heads] + [(0, 0), (B - 1, Hv - 1)]
    mp = W.model_params(wl)
    grp = Hv // Hk
    t = Tally()
    for layer in layers:
        rb_layer = oplan.layer_row_bits(layer)
        offs = oplan.layer_head_off(layer)
        nb = oplan.head_bytes[layer * Hv:(layer + 1) * Hv]
        w_layer = oplan.layer_w(layer)
        pages = {}
        states = W.random_states(wl, len(units[layer]), seed=100 + layer)
        for n, (b, h) in enumerate(units[layer]):
            page = O.encode_head(states[n], oplan.unit_kind, rb_layer[h], w_layer[h])
            base = int(slots[b]) * oplan.slot_stride + int(offs[h])
            pool[base:base + int(nb[h])] = torch.from_numpy(page).to(dev)
            pages[(b, h)] = page
        inp = W.step_inputs(wl, mp, W.STREAM_DECODE, 3, layer)
        q, k, v, beta, gate = [torch.from_numpy(x).to(dev) for x in
                               (inp.q, inp.k, inp.v, inp.beta, inp.gate)]
        y = torch.empty((B, Hv, 128), dtype=torch.float32, device=dev)
        A.stepq_decode_step(plan, layer, pool, slots_d, q, k, v, beta, gate, y)
        torch.cuda.synchronize()
        assert A.stepq_device_error() == 0
        y_h = y.cpu().numpy()
        assert np.isfinite(y_h).all()
        for (b, h), page in pages.items():
            page_o, y_o = O.step_head(page, oplan.unit_kind, rb_layer[h], w_layer[h],
                                      inp.q[b, h // grp], inp.k[b, h // grp], inp.v[b, h],
                                      inp.beta[b, h], inp.gate[b, h], wl.fit_iters)
            base = int(slots[b]) * oplan.slot_stride + int(offs[h])
            page_g = pool[base:base + int(nb[h])].cpu().numpy()
            compare_y(t, y_h[b, h], y_o)
            compare_head(t, page_g, page_o, oplan.unit_kind, rb_layer[h], w_layer[h])
    print(name, t.summary())
    t.check()
