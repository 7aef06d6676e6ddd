"""The decode step inside a CUDA graph: one step per layer captured with the
library's entry points on a capture stream, then replayed with new inputs
copied into the captured buffers. Pages and outputs must equal those of direct
calls bit for bit (the calls never synchronise or allocate, so they can be
captured)."""
import numpy as np
import pytest

from paper_2609_38169_gb300 import api as A, workloads as W

from gpu_helpers import plans

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,kw", [("pool", dict(layers=2, pool_slots=48, batch=32)), ("channel", dict(batch=16, pool_slots=24))])
def test_graph_replay_equals_direct_calls(name, kw):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    wl = W.WORKLOADS[name].replace(**kw)
    cfg, plan, oplan, _ = plans(wl)
    dev = torch.device("cuda", 0)
    B, L = wl.batch, wl.layers
    slots = torch.from_numpy(np.random.default_rng(3).permutation(wl.pool_slots)[:B].astype(np.int32)).to(dev)
    pool0 = A.alloc_pool(plan, wl.pool_slots, dev)
    all_slots = torch.arange(wl.pool_slots, dtype=torch.int32, device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    for layer in range(L):
        S = torch.randn((wl.pool_slots, wl.hv, 128, 128), generator=g, device=dev)
        A.stepq_quantize_pool(plan, layer, S, all_slots, pool0)
    mp = W.model_params_torch(W.model_params(wl), dev)
    steps = [[W.torch_step_inputs(wl, mp, t, layer, dev) for layer in range(L)] for t in range(3)]

    # direct calls
    pool_d = pool0.clone()
    y_d = []
    for t in range(3):
        ys = []
        for layer in range(L):
            y = torch.empty((B, wl.hv, 128), device=dev)
            A.stepq_decode_step(plan, layer, pool_d, slots, *steps[t][layer], y, pool_slots=wl.pool_slots)
            ys.append(y)
        y_d.append(torch.stack(ys))
    torch.cuda.synchronize()

    # one captured step, replayed three times with each step's inputs copied in
    pool_g = pool0.clone()
    ins = [[x.clone() for x in steps[0][layer]] for layer in range(L)]
    y_g = torch.empty((L, B, wl.hv, 128), device=dev)
    graph = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream(dev)
    side.wait_stream(torch.cuda.current_stream(dev))
    with torch.cuda.graph(graph, stream=side):
        for layer in range(L):
            A.stepq_decode_step(plan, layer, pool_g, slots, *ins[layer], y_g[layer],
                                pool_slots=wl.pool_slots, stream=side)
    torch.cuda.synchronize()
    # capture only records: the pool is still the initial one
    assert torch.equal(pool_g, pool0)
    for t in range(3):
        for layer in range(L):
            for dst, src in zip(ins[layer], steps[t][layer]):
                dst.copy_(src)
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(y_g, y_d[t]), t
    assert torch.equal(pool_g, pool_d)
    assert A.stepq_device_error() == 0
