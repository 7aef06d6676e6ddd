"""Shared helpers of the GPU parity tests: plans from oracle statistics, pools
moved between the oracle (numpy) and the library (torch), and the comparison
rules of the parity protocol.

Tolerances (teacher-forced, both sides start every step from the oracle's pool):
 * readout y: ||y_gpu - y_ora|| / ||y_ora|| <= 1e-4 per (slot, head), and every
   element within 1e-4 * ||y_ora||_inf;
 * integer codes: identical except +-1 LSB on at most 1e-4 of the elements
   (fp32 reduction order decides rare rounding ties);
 * FP16 row factors r: identical except 1 ulp on at most 1% of the rows (r_i
   depends on one row sum only);
 * FP16 column factors c: identical on at least 99% of the columns. A column may
   differ when a rounding tie in the first fixed-code pass (codes z0 from the
   clip-free start) fell the other way: the least-squares update then moves by
   about alpha_i (2|q|+1) / sum_i alpha_i q_i^2 per flipped code
   (alpha_i = w_i^2 r_i^2 zs_i^2), several fp16 ulps at 4 bits. Each differing
   c_j must stay within three such flips (plus one ulp);
 * FP16 pivot values: counted with the codes (a 1-ulp difference is one LSB).
"""
from __future__ import annotations

import numpy as np

import oracle as O
from paper_2609_38169_gb300 import api as A, workloads as W

Y_REL = 1e-4
CODE_FRAC = 1e-4
SCALE_FRAC = 1e-2


def plans(wl, seqs=2, steps=16):
    st = O.calibrate(wl, seqs=seqs, steps=steps)
    oplan = O.plan_from_stats(wl, st)
    cfg = A.Config.from_workload(wl)
    plan = A.stepq_fit_scales(cfg, st.omega, st.mean_log_ret, st.dist, st.pivot)
    assert np.array_equal(plan.unit_bits, oplan.unit_bits)
    assert plan.slot_stride == oplan.slot_stride
    return cfg, plan, oplan, st


def to_dev(*arrays, device="cuda"):
    import torch
    return [torch.from_numpy(np.ascontiguousarray(a)).to(device) for a in arrays]


class Tally:
    def __init__(self):
        self.elems = 0
        self.code_diff = 0
        self.code_maxdiff = 0
        self.scales = 0
        self.scale_diff = 0
        self.scale_maxulp = 0
        self.r_maxulp = 0
        self.y_worst = 0.0
        self.y_elem_worst = 0.0
        self.c_excess = 0.0          # worst |dc|/c over its allowed flip bound
        self.c_worst = ""

    def summary(self):
        return (f"codes {self.code_diff}/{self.elems} (max {self.code_maxdiff}), "
                f"scales {self.scale_diff}/{self.scales} (max {self.scale_maxulp} ulp), "
                f"y rel {self.y_worst:.2e}, y elem {self.y_elem_worst:.2e}, "
                f"c vs flip bound {self.c_excess:.2f} {self.c_worst}")

    def check(self):
        assert self.code_maxdiff <= 1, self.summary()
        assert self.code_diff <= CODE_FRAC * self.elems, self.summary()
        assert self.r_maxulp <= 1, self.summary()
        assert self.scale_diff <= SCALE_FRAC * max(self.scales, 1), self.summary()
        assert self.c_excess <= 1.0, self.summary()
        assert self.y_worst <= Y_REL, self.summary()
        assert self.y_elem_worst <= Y_REL, self.summary()


def _f16_ulps(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    """Distance in binary16 ulps between two arrays of fp16 bit patterns."""
    def ordered(u):
        u = u.astype(np.int32)
        return np.where(u & 0x8000, 0x8000 - (u & 0x7FFF), 0x8000 + u)
    return np.abs(ordered(a) - ordered(b))


def compare_head(t: Tally, page_gpu, page_ora, unit_kind, rb, w=None, piv_tol=None):
    """piv_tol: optional [128][128] absolute allowance for FP16 pivot values; a
    pivot value within it (plus one FP16 ulp of rounding) of the oracle's counts
    as equal (used where a value is the small difference of two large fp32 terms)."""
    rg, cg, zg, pg = O.unpack_head(page_gpu, unit_kind, rb)
    ro, co, zo, po = O.unpack_head(page_ora, unit_kind, rb)
    piv_rows = rb == O.PIVOT_BITS
    dz = np.abs(zg.astype(np.int32) - zo.astype(np.int32))[~piv_rows]
    dp = _f16_ulps(pg[piv_rows], po[piv_rows])
    if piv_tol is not None and piv_rows.any():
        vg = pg[piv_rows].view(np.float16).astype(np.float64)
        vo = po[piv_rows].view(np.float16).astype(np.float64)
        with np.errstate(over="ignore"):                # the spacing above 65504 is inf
            ulp = np.spacing(np.abs(po[piv_rows].view(np.float16))).astype(np.float64)
        dp = np.where(np.abs(vg - vo) <= np.asarray(piv_tol)[piv_rows] + ulp, 0, dp)
    t.elems += zg.size
    t.code_diff += int(np.count_nonzero(dz)) + int(np.count_nonzero(dp))
    t.code_maxdiff = max(t.code_maxdiff, int(dz.max(initial=0)), int(dp.max(initial=0)))
    if unit_kind == O.UNIT_HEAD and rb[0] == O.PIVOT_BITS:
        return
    ur = _f16_ulps(rg[~piv_rows], ro[~piv_rows])
    uc = _f16_ulps(cg, co)
    u = np.concatenate([ur, uc])
    t.scales += u.size
    t.scale_diff += int(np.count_nonzero(u))
    t.scale_maxulp = max(t.scale_maxulp, int(u.max(initial=0)))
    t.r_maxulp = max(t.r_maxulp, int(ur.max(initial=0)))
    if uc.any():
        w = np.ones(128) if w is None else np.asarray(w, np.float64)
        r = np.asarray(ro, np.uint16).view(np.float16).astype(np.float64)
        bits = rb.astype(np.int64)
        zs = np.where(piv_rows, 0.0, 2.0 ** (8 - np.where(piv_rows, 8, bits))) \
            if unit_kind == O.UNIT_ROW else np.ones(128)
        qm = np.where(piv_rows, 0, 2 ** (np.where(piv_rows, 2, bits) - 1) - 1)
        alpha = np.where(piv_rows, 0.0, (w * r * zs) ** 2)
        c_o = np.asarray(co, np.uint16).view(np.float16).astype(np.float64)
        c_g = np.asarray(cg, np.uint16).view(np.float16).astype(np.float64)
        for j in np.flatnonzero(uc):
            den = np.sum(alpha * zo[:, j].astype(np.float64) ** 2)
            flip = np.max(alpha * (2 * qm + 1)) / max(den, 1e-300)
            bound = 3 * flip + 2.0 ** -10
            rel = abs(c_g[j] - c_o[j]) / c_o[j]
            if rel / bound > t.c_excess:
                t.c_excess = rel / bound
                t.c_worst = (f"[col {j}: {int(uc[j])} ulp, rel {rel:.2e}, flip {flip:.2e}, "
                             f"bits {sorted(set(bits[~piv_rows].tolist()))}]")


def compare_y(t: Tally, y_gpu, y_ora):
    yg = y_gpu.reshape(-1, 128).astype(np.float64)
    yo = y_ora.reshape(-1, 128).astype(np.float64)
    nrm = np.linalg.norm(yo, axis=1)
    rel = np.linalg.norm(yg - yo, axis=1) / np.maximum(nrm, 1e-30)
    elem = np.abs(yg - yo).max(axis=1) / np.maximum(np.abs(yo).max(axis=1), 1e-30)
    t.y_worst = max(t.y_worst, float(rel.max(initial=0)))
    t.y_elem_worst = max(t.y_elem_worst, float(elem.max(initial=0)))


def compare_pools(t: Tally, pool_gpu: np.ndarray, pool_ora: np.ndarray, oplan, layer, slots,
                  units=None, piv_tol=None):
    """piv_tol: optional [B][Hv][128][128] pivot allowances (see compare_head)."""
    rbl = oplan.layer_row_bits(layer)
    offs = oplan.layer_head_off(layer)
    nb = oplan.head_bytes[layer * oplan.hv:(layer + 1) * oplan.hv]
    it = units if units is not None else [(b, h) for b in range(len(slots)) for h in range(oplan.hv)]
    for b, h in it:
        base = int(slots[b]) * oplan.slot_stride + int(offs[h])
        pg = pool_gpu[base:base + int(nb[h])]
        po = pool_ora[base:base + int(nb[h])]
        compare_head(t, pg, po, oplan.unit_kind, rbl[h], oplan.w[layer, h],
                     None if piv_tol is None else piv_tol[b, h])
