"""Seeded synthetic decode workloads for the gated Delta-rule state step.

This module only draws inputs (queries, keys, values, write strengths, gates and
the fixed per-head "model" properties that shape them). It holds none of the
quantization method's arithmetic, so both the CPU oracle and the CUDA path use it.

The paper's workloads (Qwen3.8-27B / Kimi-Linear traces on WikiText-2 and C4) are
not available; these generators stand in for them with the shapes of the paper's
hybrid models (d_k = d_v = 128, Sec. 2.1 and Table `config`) and the value
structure it reports: scalar per-head gates for GDN, per-key-channel gates for
KDA (Sec. 2.1), long-lived heads (Sec. 3.1) and per-key-row magnitude spread
(Sec. 4.2). `with_geometry` adds fixed lognormal value-channel scales (and
resizes the key-channel ones) so that the states' median max-to-median RMS
contrasts match the ones the paper measures (App. B.6: about 10x rows / 19x
columns for the GDN model, 13x / 5x for KDA).

Recipe (every draw comes from numpy's PCG64 seeded by a SeedSequence over
(seed, stream, step, layer), so any step of any layer can be drawn alone):

* q ~ N(0, 1); k = n / ||n|| per key head, n ~ N(0, 1) scaled channel-wise by
  fixed lognormal(0, k_sigma) factors per (layer, key head, channel);
  v ~ N(0, 1) scaled by fixed lognormal(0, v_sigma) factors per (layer, value
  head, channel).
* beta = sigmoid(N(0, 1)) per (slot, value head).
* scalar gate alpha ~ U(lo, hi) per (slot, value head, step); a fixed fraction of
  heads is "long-lived" with alpha ~ U(long_lo, long_hi).
* channel gate d_i = clip(base_i * exp(0.01 N(0, 1)), lo, hi), base_i ~ U(lo, hi)
  fixed per (layer, head, key channel).

Stream 0 is the decode stream, stream 1 the calibration stream, stream 2 the
warm-up that builds the initial state; the fixed model properties use stream 99.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass

import numpy as np

DK = 128
DV = 128

STREAM_DECODE = 0
STREAM_CALIB = 1
STREAM_WARMUP = 2
STREAM_MODEL = 99


@dataclass(frozen=True)
class Workload:
    name: str
    layers: int
    hk: int
    hv: int
    batch: int
    pool_slots: int
    steps: int
    gate: str                      # "scalar" (GDN, head units) or "channel" (KDA, row units)
    nominal_bits: int
    candidates: tuple
    n_pivots: int
    warmup_steps: int = 32
    alpha_lo: float = 0.90
    alpha_hi: float = 0.999
    long_frac: float = 0.0
    long_lo: float = 0.998
    long_hi: float = 0.999
    chan_lo: float = 0.80
    chan_hi: float = 0.999
    chan_jitter: float = 0.01
    k_sigma: float = 0.0           # key-channel lognormal spread (row outliers)
    v_sigma: float = 0.0           # value-channel lognormal spread (column outliers)
    calib_seqs: int = 8
    calib_steps: int = 256
    calib_every: int = 8
    horizon: int = 2048
    fit_iters: int = 1
    seed: int = 0

    @property
    def unit_kind(self) -> int:
        return 0 if self.gate == "scalar" else 1

    @property
    def gate_per_row(self) -> bool:
        return self.gate == "channel"

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads as specified: tiny decode, GQA decode, channel-gate
# decode, the 1024-slot serving pool and the long-generation drift run. q, v ~
# N(0, 1) and normalised k ~ N(0, 1); the channel-gate workloads scale the key
# channels by lognormal(0, 1) factors (a per-key-row magnitude spread).
WORKLOADS = {
    "tiny": Workload("tiny", layers=1, hk=4, hv=4, batch=1, pool_slots=1, steps=64,
                     gate="scalar", nominal_bits=6, candidates=(4, 6, 8), n_pivots=0),
    "gqa": Workload("gqa", layers=1, hk=16, hv=32, batch=64, pool_slots=64, steps=256,
                    gate="scalar", nominal_bits=6, candidates=(4, 6, 8), n_pivots=0,
                    alpha_lo=0.85, alpha_hi=0.999, long_frac=0.25),
    "channel": Workload("channel", layers=1, hk=32, hv=32, batch=256, pool_slots=256, steps=512,
                        gate="channel", nominal_bits=4, candidates=(2, 4, 6, 8), n_pivots=26,
                        k_sigma=1.0),
    "pool": Workload("pool", layers=16, hk=32, hv=32, batch=1024, pool_slots=1024, steps=128,
                     gate="scalar", nominal_bits=6, candidates=(4, 6, 8), n_pivots=7),
    "drift": Workload("drift", layers=4, hk=32, hv=32, batch=128, pool_slots=128, steps=8192,
                      gate="channel", nominal_bits=6, candidates=(4, 6, 8), n_pivots=102,
                      k_sigma=1.0),
}

# Channel spreads that give the states the outlier geometry the paper measures
# on its traces: median max-to-median RMS contrasts of about 10x along key
# rows and 19x along value columns for the GDN model, 13x and 5x for KDA
# (App. B.6), on snapshots of these recurrences from a zero state.
GDN_K_SIGMA, GDN_V_SIGMA = 1.05, 1.12
KDA_K_SIGMA, KDA_V_SIGMA = 1.10, 0.60


def with_geometry(wl: Workload) -> Workload:
    """The workload with lognormal key- and value-channel spreads sized to the
    state geometry of App. B.6 (value-column outliers included)."""
    if wl.gate == "scalar":
        return wl.replace(k_sigma=GDN_K_SIGMA, v_sigma=GDN_V_SIGMA)
    return wl.replace(k_sigma=KDA_K_SIGMA, v_sigma=KDA_V_SIGMA)


def _rng(*key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(x) for x in key])))


@dataclass
class ModelParams:
    """Fixed per-head properties of the synthetic model (shared by all streams)."""
    long_lived: np.ndarray      # [L][Hv] bool (scalar gate)
    chan_base: np.ndarray       # [L][Hv][DK] float64 (channel gate)
    k_scale: np.ndarray         # [L][Hk][DK] float64 (1 when k_sigma = 0)
    v_scale: np.ndarray         # [L][Hv][DV] float64 (1 when v_sigma = 0)


def model_params(wl: Workload) -> ModelParams:
    g = _rng(wl.seed, STREAM_MODEL)
    n_long = int(round(wl.long_frac * wl.hv))
    long_lived = np.zeros((wl.layers, wl.hv), dtype=bool)
    for layer in range(wl.layers):
        long_lived[layer, g.permutation(wl.hv)[:n_long]] = True
    chan_base = g.uniform(wl.chan_lo, wl.chan_hi, size=(wl.layers, wl.hv, DK))
    if wl.k_sigma > 0:
        k_scale = g.lognormal(0.0, wl.k_sigma, size=(wl.layers, wl.hk, DK))
    else:
        k_scale = np.ones((wl.layers, wl.hk, DK))
    if wl.v_sigma > 0:
        v_scale = g.lognormal(0.0, wl.v_sigma, size=(wl.layers, wl.hv, DV))
    else:
        v_scale = np.ones((wl.layers, wl.hv, DV))
    return ModelParams(long_lived, chan_base, k_scale, v_scale)


@dataclass
class StepInputs:
    q: np.ndarray      # [B][Hk][DK] float32
    k: np.ndarray      # [B][Hk][DK] float32, unit L2 norm
    v: np.ndarray      # [B][Hv][DV] float32
    beta: np.ndarray   # [B][Hv] float32
    gate: np.ndarray   # [B][Hv] (scalar) or [B][Hv][DK] (channel) float32


def step_inputs(wl: Workload, mp: ModelParams, stream: int, step: int, layer: int,
                batch: int | None = None) -> StepInputs:
    """Inputs of one decode step of one layer for `batch` slots."""
    b = wl.batch if batch is None else batch
    g = _rng(wl.seed, stream, step, layer)
    q = g.standard_normal((b, wl.hk, DK))
    n = g.standard_normal((b, wl.hk, DK)) * mp.k_scale[layer][None]
    k = n / np.linalg.norm(n, axis=-1, keepdims=True)
    v = g.standard_normal((b, wl.hv, DV)) * mp.v_scale[layer][None]
    beta = 1.0 / (1.0 + np.exp(-g.standard_normal((b, wl.hv))))
    if wl.gate == "scalar":
        lo = np.where(mp.long_lived[layer], wl.long_lo, wl.alpha_lo)
        hi = np.where(mp.long_lived[layer], wl.long_hi, wl.alpha_hi)
        u = g.random((b, wl.hv))
        gate = lo[None] + (hi - lo)[None] * u
    else:
        jit = np.exp(wl.chan_jitter * g.standard_normal((b, wl.hv, DK)))
        gate = np.clip(mp.chan_base[layer][None] * jit, wl.chan_lo, wl.chan_hi)
    f = np.float32
    return StepInputs(q.astype(f), k.astype(f), v.astype(f), beta.astype(f), gate.astype(f))


def slot_permutation(wl: Workload) -> np.ndarray:
    """Slot ids of the active batch: a seeded random permutation of the pool (int32)."""
    g = _rng(wl.seed, 7)
    return g.permutation(wl.pool_slots)[: wl.batch].astype(np.int32)


def random_states(wl: Workload, n: int, seed: int = 5, scale: float = 1.0) -> np.ndarray:
    """[n][DK][DV] float32 states with row and column magnitude spread (test inputs)."""
    g = _rng(wl.seed, seed)
    base = g.standard_normal((n, DK, DV))
    rows = np.exp(g.normal(0.0, 1.0, size=(n, DK, 1)))
    cols = np.exp(g.normal(0.0, 1.0, size=(n, 1, DV)))
    return (scale * base * rows * cols).astype(np.float32)


# ---- device-side draws for full-size timing runs (torch Philox; same recipe) ----

def torch_step_inputs(wl: Workload, mp_dev: dict, step: int, layer: int, device,
                      stream: int = STREAM_DECODE, batch: int | None = None):
    """Same distributions as `step_inputs`, drawn on the GPU with torch's generator.

    Used where the oracle never sees the values (timing runs). `mp_dev` holds the
    model params as device tensors: long_lived [L][Hv], chan_base [L][Hv][DK],
    k_scale [L][Hk][DK], v_scale [L][Hv][DV].
    """
    import torch
    g = torch.Generator(device=device)
    g.manual_seed((wl.seed * 1_000_003 + stream * 10_007 + step * 131 + layer) & 0x7FFF_FFFF_FFFF)
    b = wl.batch if batch is None else batch
    f = torch.float32
    q = torch.randn((b, wl.hk, DK), generator=g, device=device, dtype=f)
    n = torch.randn((b, wl.hk, DK), generator=g, device=device, dtype=f) * mp_dev["k_scale"][layer][None]
    k = n / torch.linalg.vector_norm(n, dim=-1, keepdim=True)
    v = torch.randn((b, wl.hv, DV), generator=g, device=device, dtype=f) * mp_dev["v_scale"][layer][None]
    beta = torch.sigmoid(torch.randn((b, wl.hv), generator=g, device=device, dtype=f))
    if wl.gate == "scalar":
        ll = mp_dev["long_lived"][layer]
        lo = torch.where(ll, wl.long_lo, wl.alpha_lo).to(f)
        hi = torch.where(ll, wl.long_hi, wl.alpha_hi).to(f)
        u = torch.rand((b, wl.hv), generator=g, device=device, dtype=f)
        gate = lo[None] + (hi - lo)[None] * u
    else:
        jit = torch.exp(wl.chan_jitter * torch.randn((b, wl.hv, DK), generator=g, device=device, dtype=f))
        gate = torch.clamp(mp_dev["chan_base"][layer][None] * jit, wl.chan_lo, wl.chan_hi)
    return q, k, v, beta, gate.contiguous()


def model_params_torch(mp: ModelParams, device) -> dict:
    import torch
    return {
        "long_lived": torch.as_tensor(mp.long_lived, device=device),
        "chan_base": torch.as_tensor(mp.chan_base, dtype=torch.float32, device=device),
        "k_scale": torch.as_tensor(mp.k_scale, dtype=torch.float32, device=device),
        "v_scale": torch.as_tensor(mp.v_scale, dtype=torch.float32, device=device),
    }
