"""Chunked prefill on FP32 states (the uncompressed side of the prefill
boundary) against the oracle's token-by-token recurrence, and the boundary
itself: prefill, then pack with stepq_quantize_pool."""
import numpy as np
import pytest

import oracle as O
from paper_2609_38169_gb300 import api as A, workloads as W

from gpu_helpers import Tally, compare_pools, plans, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as T
    if not T.cuda.is_available():
        pytest.skip("no CUDA device")
    return T


def _tokens(wl, B, T, layer=0):
    mp = W.model_params(wl)
    steps = [W.step_inputs(wl, mp, W.STREAM_DECODE, t, layer, batch=B) for t in range(T)]
    stack = lambda f: np.ascontiguousarray(np.stack([f(s) for s in steps], axis=1))
    return (stack(lambda s: s.q), stack(lambda s: s.k), stack(lambda s: s.v),
            stack(lambda s: s.beta), stack(lambda s: s.gate))


def _reference(S0, q, k, v, beta, gate):
    S = S0.copy()
    ys = [O.delta_batch(S, q[:, t], k[:, t], v[:, t], beta[:, t], gate[:, t]) for t in range(q.shape[1])]
    return S, np.stack(ys, axis=1)


@pytest.mark.parametrize("name,T", [("gqa", 70), ("gqa", 32), ("gqa", 5), ("channel", 40), ("tiny", 64)])
def test_prefill_matches_recurrence(torch, name, T):
    """Eq. delta_update over T tokens, chunked by 32 (full chunks and a ragged tail)."""
    wl = W.WORKLOADS[name]
    B = 2
    cfg = A.Config.from_workload(wl)
    S0 = O.warmup_states(wl, 0, B)
    q, k, v, beta, gate = _tokens(wl, B, T)
    S_o, y_o = _reference(S0, q, k, v, beta, gate)
    S_d, q_d, k_d, v_d, b_d, g_d = to_dev(S0, q, k, v, beta, gate)
    y_d = torch.empty((B, T, wl.hv, 128), dtype=torch.float32, device="cuda")
    A.stepq_prefill_fp32(cfg, S_d, q_d, k_d, v_d, b_d, g_d, y_d)
    y_g, S_g = y_d.cpu().numpy(), S_d.cpu().numpy()
    rel = np.linalg.norm(y_g - y_o, axis=-1) / np.maximum(np.linalg.norm(y_o, axis=-1), 1e-30)
    assert rel.max() <= 1e-4, rel.max()
    assert np.abs(S_g - S_o).max() <= 1e-4 * np.abs(S_o).max()


@pytest.mark.parametrize("name,B,T", [("gqa", 10, 45), ("channel", 6, 33)])
def test_prefill_several_items_per_cta(torch, name, B, T):
    """More (slot, head) items than SMs, so that each persistent CTA prepares the
    next item's first chunk while the previous item's last chunk finishes; the
    ragged tails end every item."""
    wl = W.WORKLOADS[name]
    cfg = A.Config.from_workload(wl)
    assert B * wl.hv > torch.cuda.get_device_properties(0).multi_processor_count
    S0 = O.warmup_states(wl, 0, B)
    q, k, v, beta, gate = _tokens(wl, B, T)
    S_o, y_o = _reference(S0, q, k, v, beta, gate)
    S_d, q_d, k_d, v_d, b_d, g_d = to_dev(S0, q, k, v, beta, gate)
    y_d = torch.empty((B, T, wl.hv, 128), dtype=torch.float32, device="cuda")
    A.stepq_prefill_fp32(cfg, S_d, q_d, k_d, v_d, b_d, g_d, y_d)
    y_g, S_g = y_d.cpu().numpy(), S_d.cpu().numpy()
    rel = np.linalg.norm(y_g - y_o, axis=-1) / np.maximum(np.linalg.norm(y_o, axis=-1), 1e-30)
    assert rel.max() <= 1e-4, rel.max()
    assert np.abs(S_g - S_o).max() <= 1e-4 * np.abs(S_o).max()
    assert A.stepq_device_error() == 0


def test_prefill_empty_and_identity(torch):
    """T = 0 is a no-op; beta = 0 with gate 1 leaves the state unchanged."""
    wl = W.WORKLOADS["tiny"]
    cfg = A.Config.from_workload(wl)
    S0 = O.warmup_states(wl, 0, 1)
    q, k, v, beta, gate = _tokens(wl, 1, 33)
    S_d, q_d, k_d, v_d = to_dev(S0, q, k, v)
    b_d, g_d = to_dev(np.zeros_like(beta), np.ones_like(gate))
    y_d = torch.empty((1, 33, wl.hv, 128), dtype=torch.float32, device="cuda")
    A.stepq_prefill_fp32(cfg, S_d, q_d[:, :0].contiguous(), k_d[:, :0].contiguous(),
                         v_d[:, :0].contiguous(), b_d[:, :0].contiguous(), g_d[:, :0].contiguous(),
                         y_d[:, :0].contiguous())
    assert np.array_equal(S_d.cpu().numpy(), S0)
    A.stepq_prefill_fp32(cfg, S_d, q_d, k_d, v_d, b_d, g_d, y_d)
    assert np.abs(S_d.cpu().numpy() - S0).max() <= 1e-6 * np.abs(S0).max()
    # y_t = S0^T q_t for every token
    y_o = np.einsum("bhij,bthi->bthj", S0.astype(np.float64), np.repeat(q, 1, axis=2))
    rel = np.linalg.norm(y_d.cpu().numpy() - y_o, axis=-1) / np.linalg.norm(y_o, axis=-1)
    assert rel.max() <= 1e-5


@pytest.mark.parametrize("name", ["gqa", "channel"])
def test_prefill_boundary_packs_like_the_oracle(torch, name):
    """Prefill from a stored state (unpack), then pack the boundary state.

    The unpacked start is the oracle's decode exactly; the prefilled state is
    within 1e-4 of the oracle's token-by-token recurrence; and the page packed
    on the device matches the oracle's encoding of that same prefilled state
    (the same-input parity bar: codes +-1 LSB on at most 1e-4 of elements).
    The page is not compared with the oracle's encoding of its own prefilled
    state: the two states differ by fp32 rounding, and in low-magnitude rows
    (the key-row and value-column outliers give them steps far below 1e-4 of
    the state's maximum) that difference alone can move a code by several
    levels."""
    wl = W.WORKLOADS[name]
    B, T = 4, 48
    cfg, plan, oplan, _ = plans(wl)
    slots = np.array([3, 0, 7, 5], np.int32)[:B]
    pool_o = np.zeros(wl.pool_slots * oplan.slot_stride, np.uint8)
    O.pool_encode(oplan, pool_o, 0, slots, O.warmup_states(wl, 0, B))
    S_start = O.pool_decode(oplan, pool_o, 0, slots).astype(np.float32)
    q, k, v, beta, gate = _tokens(wl, B, T)
    S_o, _ = _reference(S_start, q, k, v, beta, gate)
    (slots_d,) = to_dev(slots)
    pool_d = torch.from_numpy(pool_o).cuda()
    states = torch.empty((B, wl.hv, 128, 128), dtype=torch.float32, device="cuda")
    A.stepq_dequantize_pool(plan, 0, pool_d, slots_d, states)
    assert np.array_equal(states.cpu().numpy(), S_start)
    q_d, k_d, v_d, b_d, g_d = to_dev(q, k, v, beta, gate)
    y_d = torch.empty((B, T, wl.hv, 128), dtype=torch.float32, device="cuda")
    A.stepq_prefill_fp32(cfg, states, q_d, k_d, v_d, b_d, g_d, y_d)
    S_g = states.cpu().numpy()
    assert np.abs(S_g - S_o).max() <= 1e-4 * np.abs(S_o).max()
    A.stepq_quantize_pool(plan, 0, states, slots_d, pool_d)
    pool_ref = pool_o.copy()
    O.pool_encode(oplan, pool_ref, 0, slots, S_g)
    t = Tally()
    compare_pools(t, pool_d.cpu().numpy(), pool_ref, oplan, 0, slots)
    print(name, t.summary())
    t.check()
