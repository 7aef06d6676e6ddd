"""STEPQuant CPU oracle — TEST INFRASTRUCTURE ONLY.

A plain, slow restatement of the paper's method in C (fp64, scalar loops; see
oracle.h for the precision contract and the readings it takes), with this thin
ctypes/numpy wrapper. Only `tests/`, `__graft_entry__.smoke()` and the CPU
baseline leg of `bench.py` may import it. It shares no code with the CUDA
library; the two meet only through the seeded input generators in
`paper_2609_38169_gb300.workloads`.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")
_SOURCES = ["numerics.c", "recurrence.c", "codec.c", "plan.c", "batch.c", "calib.c"]

UNIT_HEAD = 0
UNIT_ROW = 1
PIVOT_BITS = 16
D = 128


def build(force: bool = False) -> str:
    """Compile liboracle.so with gcc (plain C11, -O2, OpenMP, no FP contraction)."""
    srcs = [os.path.join(_HERE, s) for s in _SOURCES] + [os.path.join(_HERE, "oracle.h")]
    if not force and os.path.exists(_SO):
        so_t = os.path.getmtime(_SO)
        if all(os.path.getmtime(s) <= so_t for s in srcs):
            return _SO
    os.makedirs(_BUILD, exist_ok=True)
    tmp = _SO + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
           "-Wall", "-o", tmp] + [os.path.join(_HERE, s) for s in _SOURCES] + ["-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


_lib = None


def lib():
    global _lib
    if _lib is None:
        # STEPQ_ORACLE_LIB names a separately built copy of this library; the
        # planted-mistake tests (tests/test_oracle_mutations.py) run the pins
        # against mutated copies this way.
        path = os.environ.get("STEPQ_ORACLE_LIB")
        _lib = C.CDLL(path if path else build())
        _declare(_lib)
    return _lib


P = C.c_void_p
I = C.c_int
D_ = C.c_double
F = C.c_float
U64 = C.c_uint64
LL = C.c_longlong


def _declare(L):
    sig = {
        "or_fp16_round": (D_, [D_]),
        "or_fp16_encode": (C.c_uint16, [D_]),
        "or_fp16_decode": (D_, [C.c_uint16]),
        "or_delta_step_f32": (None, [P, P, P, P, F, P, I, P]),
        "or_delta_batch_f32": (None, [I, I, I, I, P, P, P, P, P, P, P]),
        "or_delta_step_read_f32": (None, [P, P, P, P, P, F, P, I, P]),
        "or_delta_batch_read_f32": (None, [I, I, I, I, P, P, P, P, P, P, P, P]),
        "or_row_impact": (None, [P, P, F, P, I, P]),
        "or_row_impact_dense": (None, [P, P, F, P, I, P]),
        "or_head_bytes": (C.c_size_t, [I, P]),
        "or_encode_head": (None, [P, I, P, P, I, P]),
        "or_decode_head": (None, [P, I, P, P]),
        "or_decode_head_f32": (None, [P, I, P, P]),
        "or_step_head": (None, [P, I, P, P, I, P, P, P, F, P, I, P, P]),
        "or_unpack_head": (None, [P, I, P, P, P, P, P]),
        "or_fit_debug": (None, [P, I, P, P, I, P, P, P]),
        "or_intb_head_bytes": (C.c_size_t, [I]),
        "or_intb_encode_head": (None, [P, I, P]),
        "or_intb_decode_head": (None, [P, I, P]),
        "or_intb_step_head": (None, [P, I, P, P, P, F, P, I, P]),
        "or_temporal_head_bytes": (C.c_size_t, [P]),
        "or_temporal_encode_head": (None, [P, P, P]),
        "or_temporal_decode_head": (None, [P, P, P]),
        "or_row_weights": (None, [I, P, P]),
        "or_lifetime_weight": (D_, [D_, I]),
        "or_allocate_dp": (I, [I, I, P, LL, P, P]),
        "or_allocate_lagrangian": (I, [I, I, P, LL, P, P]),
        "or_lagrangian_multiplier": (D_, [I, I, P, LL, P]),
        "or_select_pivots": (I, [I, I, I, P, I, P, P, I, P]),
        "or_allocate": (I, [I, I, I, P, I, P, P, P, P]),
        "or_layout": (I, [I, I, I, P, P, P, P]),
        "or_pool_encode": (None, [I, I, P, P, I, P, U64, P, P, I, P]),
        "or_pool_decode": (None, [I, I, P, P, U64, P, P, I, P]),
        "or_pool_step": (None, [I, I, I, I, P, P, I, P, U64, P, P, I, P, P, P, P, P, P, P]),
        "or_pool_step_units": (None, [I, I, I, I, P, P, I, P, U64, P, P, I, P, P, P, P, P, P, P, P]),
        "or_intb_pool_step": (None, [I, I, I, I, U64, U64, P, P, I, P, P, P, P, P, P]),
        "or_calib_observe": (None, [I, I, I, I, P, P, P, P, P, P]),
        "or_calib_distortion": (None, [I, I, I, P, P, I, P, P, I, P]),
        "or_num_threads": (I, []),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args


class _Ptr(C.c_void_p):
    """A pointer argument that keeps its numpy array alive until the call returns."""
    __slots__ = ("_keep",)


def _p(a: np.ndarray | None):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"], "oracle arrays must be C-contiguous"
    ptr = _Ptr(a.ctypes.data)
    ptr._keep = a
    return ptr


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


def _i8(a):
    return np.ascontiguousarray(a, dtype=np.int8)


def num_threads() -> int:
    return lib().or_num_threads()


# ------------------------------------------------------------------ numerics
def fp16_round(x: float) -> float:
    return lib().or_fp16_round(float(x))


def fp16_encode(x: float) -> int:
    return lib().or_fp16_encode(float(x))


def fp16_decode(h: int) -> float:
    return lib().or_fp16_decode(int(h))


# --------------------------------------------------------------- recurrence
def delta_step(S, q, k, v, beta, gate):
    """One FP32-state step of one head; returns (S_new, y)."""
    S = _f32(S).copy()
    gate = _f32(np.atleast_1d(gate))
    y = np.zeros(D, np.float32)
    lib().or_delta_step_f32(_p(S), _p(_f32(q)), _p(_f32(k)), _p(_f32(v)), float(beta),
                            _p(gate), int(gate.size == D), _p(y))
    return S, y


def delta_batch(S, q, k, v, beta, gate):
    """In-place FP32-state step of S [n][Hv][128][128]; returns y [n][Hv][128]."""
    assert S.dtype == np.float32 and S.flags["C_CONTIGUOUS"]
    n, Hv = S.shape[:2]
    Hk = q.shape[1]
    gate = _f32(gate)
    y = np.zeros((n, Hv, D), np.float32)
    lib().or_delta_batch_f32(n, Hk, Hv, int(gate.ndim == 3), _p(S), _p(_f32(q)), _p(_f32(k)),
                             _p(_f32(v)), _p(_f32(beta)), _p(gate), _p(y))
    return y


def delta_step_read(S, S_ref, q, k, v, beta, gate):
    """Exact-read step of one head (App. B.1): the Delta residual reads the
    reference state, u = k^T D S_ref; returns (S_new, y)."""
    S = _f32(S).copy()
    gate = _f32(np.atleast_1d(gate))
    y = np.zeros(D, np.float32)
    lib().or_delta_step_read_f32(_p(S), _p(_f32(S_ref)), _p(_f32(q)), _p(_f32(k)), _p(_f32(v)),
                                 float(beta), _p(gate), int(gate.size == D), _p(y))
    return S, y


def delta_batch_read(S, S_ref, q, k, v, beta, gate):
    """In-place exact-read step of S [n][Hv][128][128] reading S_ref (same
    shape); returns y [n][Hv][128]."""
    assert S.dtype == np.float32 and S.flags["C_CONTIGUOUS"] and S_ref.shape == S.shape
    n, Hv = S.shape[:2]
    Hk = q.shape[1]
    gate = _f32(gate)
    y = np.zeros((n, Hv, D), np.float32)
    lib().or_delta_batch_read_f32(n, Hk, Hv, int(gate.ndim == 3), _p(S), _p(_f32(S_ref)),
                                  _p(_f32(q)), _p(_f32(k)), _p(_f32(v)), _p(_f32(beta)),
                                  _p(gate), _p(y))
    return y


def row_impact(q, k, beta, gate, dense=False):
    gate = _f32(np.atleast_1d(gate))
    g = np.zeros(D, np.float64)
    fn = lib().or_row_impact_dense if dense else lib().or_row_impact
    fn(_p(_f32(q)), _p(_f32(k)), float(beta), _p(gate), int(gate.size == D), _p(g))
    return g


# -------------------------------------------------------------------- codec
def head_row_bits(unit_kind: int, bits) -> np.ndarray:
    """Per-row widths of one head: a head unit repeats its width."""
    if unit_kind == UNIT_HEAD:
        return np.full(D, int(bits), np.int8)
    return _i8(bits)


def head_bytes(unit_kind, rb) -> int:
    return lib().or_head_bytes(unit_kind, _p(_i8(rb)))


def encode_head(X, unit_kind, rb, w, fit_iters=1) -> np.ndarray:
    rb = _i8(rb)
    page = np.zeros(head_bytes(unit_kind, rb), np.uint8)
    lib().or_encode_head(_p(_f32(X)), unit_kind, _p(rb), _p(_f32(w)), fit_iters, _p(page))
    return page


def decode_head(page, unit_kind, rb) -> np.ndarray:
    S = np.zeros((D, D), np.float64)
    lib().or_decode_head(_p(np.ascontiguousarray(page, np.uint8)), unit_kind, _p(_i8(rb)), _p(S))
    return S


def decode_head_f32(page, unit_kind, rb) -> np.ndarray:
    S = np.zeros((D, D), np.float32)
    lib().or_decode_head_f32(_p(np.ascontiguousarray(page, np.uint8)), unit_kind, _p(_i8(rb)),
                             _p(S))
    return S


def unpack_head(page, unit_kind, rb):
    r = np.zeros(D, np.uint16)
    c = np.zeros(D, np.uint16)
    codes = np.zeros((D, D), np.int8)
    piv = np.zeros((D, D), np.uint16)
    lib().or_unpack_head(_p(np.ascontiguousarray(page, np.uint8)), unit_kind, _p(_i8(rb)),
                         _p(r), _p(c), _p(codes), _p(piv))
    return r, c, codes, piv


def fit_debug(X, unit_kind, rb, w, fit_iters=1):
    """(r values, last column iterate (exact, before FP16 rounding), codes of the
    last fixed-code update)."""
    r = np.zeros(D, np.float64)
    c = np.zeros(D, np.float64)
    z = np.zeros((D, D), np.int8)
    lib().or_fit_debug(_p(_f32(X)), unit_kind, _p(_i8(rb)), _p(_f32(w)), fit_iters, _p(r), _p(c),
                       _p(z))
    return r, c, z


def step_head(page, unit_kind, rb, w, q, k, v, beta, gate, fit_iters=1):
    """One persistent decode step of a packed head; returns (new_page, y)."""
    page = np.ascontiguousarray(page, np.uint8).copy()
    gate = _f32(np.atleast_1d(gate))
    y = np.zeros(D, np.float32)
    lib().or_step_head(_p(page), unit_kind, _p(_i8(rb)), _p(_f32(w)), fit_iters, _p(_f32(q)),
                       _p(_f32(k)), _p(_f32(v)), float(beta), _p(gate), int(gate.size == D),
                       _p(y), None)
    return page, y


def intb_head_bytes(bits) -> int:
    return lib().or_intb_head_bytes(bits)


def intb_encode_head(X, bits) -> np.ndarray:
    page = np.zeros(intb_head_bytes(bits), np.uint8)
    lib().or_intb_encode_head(_p(_f32(X)), bits, _p(page))
    return page


def intb_decode_head(page, bits) -> np.ndarray:
    S = np.zeros((D, D), np.float64)
    lib().or_intb_decode_head(_p(np.ascontiguousarray(page, np.uint8)), bits, _p(S))
    return S


def intb_step_head(page, bits, q, k, v, beta, gate):
    page = np.ascontiguousarray(page, np.uint8).copy()
    gate = _f32(np.atleast_1d(gate))
    y = np.zeros(D, np.float32)
    lib().or_intb_step_head(_p(page), bits, _p(_f32(q)), _p(_f32(k)), _p(_f32(v)), float(beta),
                            _p(gate), int(gate.size == D), _p(y))
    return page, y


# --------------------------------------------------------------------- plan
def temporal_head_bytes(rb) -> int:
    return lib().or_temporal_head_bytes(_p(_i8(rb)))


def temporal_encode_head(X, rb) -> np.ndarray:
    """"Temporal only" ablation codec (Sec. 5.4): the plan's row widths rb (16 =
    FP16 pivot) with the rowwise absmax quantizer of App. B.5."""
    rb = _i8(rb)
    page = np.zeros(temporal_head_bytes(rb), np.uint8)
    lib().or_temporal_encode_head(_p(_f32(X)), _p(rb), _p(page))
    return page


def temporal_decode_head(page, rb) -> np.ndarray:
    S = np.zeros((D, D), np.float64)
    lib().or_temporal_decode_head(_p(np.ascontiguousarray(page, np.uint8)), _p(_i8(rb)), _p(S))
    return S


def row_weights(omega) -> np.ndarray:
    om = _f32(omega)
    w = np.zeros_like(om)
    lib().or_row_weights(om.size // D, _p(om), _p(w))
    return w


def lifetime_weight(ell: float, H: int) -> float:
    return lib().or_lifetime_weight(float(ell), int(H))


def allocate_dp(cost, cands, capacity_half_bits):
    cost = np.ascontiguousarray(cost, np.float64)
    U, K = cost.shape
    ch = np.zeros(U, np.int8)
    c = np.ascontiguousarray(cands, np.int32)
    rc = lib().or_allocate_dp(U, K, _p(c), int(capacity_half_bits), _p(cost), _p(ch))
    return None if rc else ch


def allocate_lagrangian(cost, cands, budget_bits):
    cost = np.ascontiguousarray(cost, np.float64)
    U, K = cost.shape
    ch = np.zeros(U, np.int8)
    c = np.ascontiguousarray(cands, np.int32)
    rc = lib().or_allocate_lagrangian(U, K, _p(c), int(budget_bits), _p(cost), _p(ch))
    return None if rc else ch


def lagrangian_multiplier(cost, cands, budget_bits):
    """The Lagrangian relaxation's multiplier (None if nothing fits)."""
    cost = np.ascontiguousarray(cost, np.float64)
    U, K = cost.shape
    c = np.ascontiguousarray(cands, np.int32)
    lam = lib().or_lagrangian_multiplier(U, K, _p(c), int(budget_bits), _p(cost))
    return None if lam < 0 else lam


def select_pivots(unit_kind, cands, nominal, L, dist, n_pivots):
    dist = np.ascontiguousarray(dist, np.float64)
    U = dist.shape[0]
    piv = np.zeros(U, np.uint8)
    c = np.ascontiguousarray(cands, np.int32)
    rc = lib().or_select_pivots(unit_kind, U, len(cands), _p(c), nominal,
                                _p(np.ascontiguousarray(L, np.float64)), _p(dist), n_pivots,
                                _p(piv))
    if rc:
        raise ValueError("pivot selection failed")
    return piv


def allocate(unit_kind, cands, nominal, L, dist, pivot):
    dist = np.ascontiguousarray(dist, np.float64)
    U = dist.shape[0]
    bits = np.zeros(U, np.int8)
    c = np.ascontiguousarray(cands, np.int32)
    rc = lib().or_allocate(unit_kind, U, len(cands), _p(c), nominal,
                           _p(np.ascontiguousarray(L, np.float64)), _p(dist),
                           _p(np.ascontiguousarray(pivot, np.uint8)), _p(bits))
    if rc:
        raise ValueError("allocation infeasible for the budget")
    return bits


def layout(unit_kind, n_layers, Hv, unit_bits):
    ub = _i8(unit_bits)
    off = np.zeros(n_layers * Hv, np.uint64)
    nb = np.zeros(n_layers * Hv, np.uint32)
    stride = np.zeros(1, np.uint64)
    lib().or_layout(unit_kind, n_layers, Hv, _p(ub), _p(off), _p(nb), _p(stride))
    return off, nb, int(stride[0])


@dataclass
class OraclePlan:
    unit_kind: int
    n_layers: int
    hk: int
    hv: int
    nominal: int
    cands: tuple
    fit_iters: int
    w: np.ndarray            # [L][Hv][128] float32
    L: np.ndarray            # [units] float64 lifetime weights
    pivot: np.ndarray        # [units] uint8
    unit_bits: np.ndarray    # [units] int8 (16 = FP16 pivot)
    head_off: np.ndarray     # [L*Hv] uint64
    head_bytes: np.ndarray   # [L*Hv] uint32
    slot_stride: int

    @property
    def gate_per_row(self) -> bool:
        return self.unit_kind == UNIT_ROW

    def layer_row_bits(self, layer: int) -> np.ndarray:
        Hv = self.hv
        if self.unit_kind == UNIT_HEAD:
            ub = self.unit_bits[layer * Hv:(layer + 1) * Hv]
            return np.repeat(ub[:, None], D, axis=1).astype(np.int8).copy()
        return self.unit_bits.reshape(self.n_layers, Hv, D)[layer].copy()

    def layer_w(self, layer: int) -> np.ndarray:
        return np.ascontiguousarray(self.w[layer], np.float32)

    def layer_head_off(self, layer: int) -> np.ndarray:
        return np.ascontiguousarray(self.head_off[layer * self.hv:(layer + 1) * self.hv])


def make_plan(unit_kind, n_layers, hk, hv, nominal, cands, n_pivots, horizon, fit_iters,
              omega, mean_log_ret, dist, pivot=None) -> OraclePlan:
    """Plan from calibration statistics: w, L, pivots (unless given), widths, layout."""
    w = row_weights(np.asarray(omega, np.float32).reshape(-1, D)).reshape(n_layers, hv, D)
    ell = np.asarray(mean_log_ret, np.float64).ravel()
    L = np.array([lifetime_weight(e, horizon) for e in ell])
    if pivot is None:
        pivot = select_pivots(unit_kind, cands, nominal, L, dist, n_pivots)
    bits = allocate(unit_kind, cands, nominal, L, dist, pivot)
    off, nb, stride = layout(unit_kind, n_layers, hv, bits)
    return OraclePlan(unit_kind, n_layers, hk, hv, nominal, tuple(cands), fit_iters, w, L,
                      np.asarray(pivot, np.uint8), bits, off, nb, stride)


# --------------------------------------------------------------------- pool
def pool_encode(plan: OraclePlan, pool: np.ndarray, layer: int, slots, states):
    slots = np.ascontiguousarray(slots, np.int32)
    lib().or_pool_encode(plan.unit_kind, plan.hv, _p(plan.layer_row_bits(layer)),
                         _p(plan.layer_w(layer)), plan.fit_iters, _p(plan.layer_head_off(layer)),
                         plan.slot_stride, _p(pool), _p(slots), len(slots), _p(_f32(states)))


def pool_decode(plan: OraclePlan, pool: np.ndarray, layer: int, slots) -> np.ndarray:
    slots = np.ascontiguousarray(slots, np.int32)
    out = np.zeros((len(slots), plan.hv, D, D), np.float32)
    lib().or_pool_decode(plan.unit_kind, plan.hv, _p(plan.layer_row_bits(layer)),
                         _p(plan.layer_head_off(layer)), plan.slot_stride, _p(pool), _p(slots),
                         len(slots), _p(out))
    return out


def pool_step(plan: OraclePlan, pool: np.ndarray, layer: int, slots, inp, with_delta=False):
    """One decode step of every (slot, head) of the layer in place; returns y, or
    (y, delta) with delta_j = v_j - k^T D S_hat (fp64) when asked."""
    slots = np.ascontiguousarray(slots, np.int32)
    B = len(slots)
    y = np.zeros((B, plan.hv, D), np.float32)
    delta = np.zeros((B, plan.hv, D), np.float64) if with_delta else None
    lib().or_pool_step(plan.unit_kind, plan.hk, plan.hv, int(plan.gate_per_row),
                       _p(plan.layer_row_bits(layer)), _p(plan.layer_w(layer)), plan.fit_iters,
                       _p(plan.layer_head_off(layer)), plan.slot_stride, _p(pool), _p(slots), B,
                       _p(_f32(inp.q)), _p(_f32(inp.k)), _p(_f32(inp.v)), _p(_f32(inp.beta)),
                       _p(_f32(inp.gate)), _p(y), _p(delta) if with_delta else None)
    return (y, delta) if with_delta else y


def pool_step_units(plan: OraclePlan, pool, layer, slots, inp, unit_b, unit_h) -> np.ndarray:
    """Step only the listed (batch index, head) units; y has the full [B][Hv][128] shape."""
    slots = np.ascontiguousarray(slots, np.int32)
    ub = np.ascontiguousarray(unit_b, np.int32)
    uh = np.ascontiguousarray(unit_h, np.int32)
    y = np.zeros((len(slots), plan.hv, D), np.float32)
    lib().or_pool_step_units(plan.unit_kind, plan.hk, plan.hv, int(plan.gate_per_row),
                             _p(plan.layer_row_bits(layer)), _p(plan.layer_w(layer)),
                             plan.fit_iters, _p(plan.layer_head_off(layer)), plan.slot_stride,
                             _p(pool), _p(slots), len(ub), _p(ub), _p(uh), _p(_f32(inp.q)),
                             _p(_f32(inp.k)), _p(_f32(inp.v)), _p(_f32(inp.beta)),
                             _p(_f32(inp.gate)), _p(y))
    return y


def intb_pool_step(bits, hk, hv, gate_per_row, layer_off, slot_stride, pool, slots, inp):
    slots = np.ascontiguousarray(slots, np.int32)
    y = np.zeros((len(slots), hv, D), np.float32)
    lib().or_intb_pool_step(bits, hk, hv, int(gate_per_row), int(layer_off), int(slot_stride),
                            _p(pool), _p(slots), len(slots), _p(_f32(inp.q)), _p(_f32(inp.k)),
                            _p(_f32(inp.v)), _p(_f32(inp.beta)), _p(_f32(inp.gate)), _p(y))
    return y


# -------------------------------------------------------------- calibration
def calib_observe(inp, omega_sum, logret_sum):
    n, Hk = inp.q.shape[:2]
    Hv = inp.v.shape[1]
    lib().or_calib_observe(n, Hk, Hv, int(inp.gate.ndim == 3), _p(_f32(inp.q)), _p(_f32(inp.k)),
                           _p(_f32(inp.beta)), _p(_f32(inp.gate)), _p(omega_sum), _p(logret_sum))


def calib_distortion(unit_kind, states, w_layer, cands, pivot_rows_layer, fit_iters, acc):
    n, Hv = states.shape[:2]
    c = np.ascontiguousarray(cands, np.int32)
    pr = None if pivot_rows_layer is None else np.ascontiguousarray(pivot_rows_layer, np.uint8)
    lib().or_calib_distortion(n, Hv, unit_kind, _p(_f32(states)), _p(_f32(w_layer)), len(cands),
                              _p(c), _p(pr), fit_iters, _p(acc))


@dataclass
class CalibStats:
    omega: np.ndarray         # [L][Hv][128] float32
    mean_log_ret: np.ndarray  # [units] float64
    dist_stage1: np.ndarray   # [units][K+1] float64 (no pivots)
    dist: np.ndarray          # [units][K+1] float64 (pivot rows excluded; = stage1 for heads)
    pivot: np.ndarray         # [units] uint8


def calibrate(wl, seqs=None, steps=None, every=None) -> CalibStats:
    """Calibration on the seeded calibration stream (App. A.3; App. C.2).

    Pass A accumulates omega and ell from the inputs; pass B replays the
    FP32-state recurrence from zero and measures candidate distortions on
    states sampled every `every` updates (each sequence a separate sample);
    row units then fix their pivots and re-measure with those rows excluded.
    """
    from paper_2609_38169_gb300 import workloads as W
    seqs = wl.calib_seqs if seqs is None else seqs
    steps = wl.calib_steps if steps is None else steps
    every = wl.calib_every if every is None else every
    mp = W.model_params(wl)
    unit_kind = wl.unit_kind
    Lyr, Hv, Hk = wl.layers, wl.hv, wl.hk
    cands = list(wl.candidates)
    K = len(cands)
    omega_sum = np.zeros((Lyr, Hv, D), np.float64)
    lr_shape = (Lyr, Hv, D) if unit_kind == UNIT_ROW else (Lyr, Hv)
    logret_sum = np.zeros(lr_shape, np.float64)
    for t in range(steps):
        for layer in range(Lyr):
            inp = W.step_inputs(wl, mp, W.STREAM_CALIB, t, layer, batch=seqs)
            calib_observe(inp, omega_sum[layer], logret_sum[layer])
    n_tok = seqs * steps
    omega = (omega_sum / n_tok).astype(np.float32)
    mean_log_ret = (logret_sum / n_tok).ravel()
    w = row_weights(omega.reshape(-1, D)).reshape(Lyr, Hv, D)

    def distortion_pass(pivot_rows):
        n_units = Lyr * Hv * (D if unit_kind == UNIT_ROW else 1)
        acc = np.zeros((Lyr, Hv * (D if unit_kind == UNIT_ROW else 1), K + 1), np.float64)
        n_samp = 0
        for layer in range(Lyr):
            S = np.zeros((seqs, Hv, D, D), np.float32)
            for t in range(steps):
                inp = W.step_inputs(wl, mp, W.STREAM_CALIB, t, layer, batch=seqs)
                delta_batch(S, inp.q, inp.k, inp.v, inp.beta, inp.gate)
                if (t + 1) % every == 0:
                    pr = None if pivot_rows is None else pivot_rows.reshape(Lyr, Hv, D)[layer]
                    calib_distortion(unit_kind, S, w[layer], cands, pr, wl.fit_iters, acc[layer])
                    if layer == 0:
                        n_samp += seqs
        return (acc / max(n_samp, 1)).reshape(n_units, K + 1)

    d1 = distortion_pass(None)
    Lw = np.array([lifetime_weight(e, wl.horizon) for e in mean_log_ret])
    pivot = select_pivots(unit_kind, cands, wl.nominal_bits, Lw, d1, wl.n_pivots)
    if unit_kind == UNIT_ROW and pivot.any():
        d2 = distortion_pass(pivot)
    else:
        d2 = d1
    return CalibStats(omega, mean_log_ret, d1, d2, pivot)


def plan_from_stats(wl, st: CalibStats) -> OraclePlan:
    return make_plan(wl.unit_kind, wl.layers, wl.hk, wl.hv, wl.nominal_bits, wl.candidates,
                     wl.n_pivots, wl.horizon, wl.fit_iters, st.omega, st.mean_log_ret, st.dist,
                     pivot=st.pivot)


def warmup_states(wl, layer: int, batch: int, steps: int | None = None) -> np.ndarray:
    """FP32-state warm-up from zero on the warm-up stream: [batch][Hv][128][128]."""
    from paper_2609_38169_gb300 import workloads as W
    steps = wl.warmup_steps if steps is None else steps
    mp = W.model_params(wl)
    S = np.zeros((batch, wl.hv, D, D), np.float32)
    for t in range(steps):
        inp = W.step_inputs(wl, mp, W.STREAM_WARMUP, t, layer, batch=batch)
        delta_batch(S, inp.q, inp.k, inp.v, inp.beta, inp.gate)
    return S
