"""Pins of the oracle's offline plan: row-impact factors (Sec. 4.3 footnote),
lifetime weights (Eq. calibration_lifetime), the allocation optimisers
(Eq. allocation, App. C.2), FP16 pivots and the packed byte counts the paper
prints (App. D, App. F.1; fixtures in tests/golden/storage.json).
"""
import itertools
import json
import os

import numpy as np
import pytest

D = 128
HEAD, ROW = 0, 1
GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "storage.json")))


def test_row_weights_geometric_mean_and_ratios(oracle, rng):
    omega = np.exp(rng.normal(0, 3, (3, D))).astype(np.float32)
    w = oracle.row_weights(omega)
    for h in range(3):
        assert abs(np.mean(np.log(w[h].astype(np.float64)))) < 1e-6       # GM(w) = 1
        i, k = rng.choice(D, 2, replace=False)
        ratio = (w[h, i] / w[h, k]).astype(np.float64) ** 8                 # w ~ omega^(gamma/2)
        assert abs(ratio / (omega[h, i] / omega[h, k]) - 1) < 1e-5


def test_lifetime_weight_closed_form(oracle):
    for ell in (-0.5, -0.05, -1e-3, -1e-6):
        for H in (1, 7, 2048):
            ref = (1 - np.exp(2 * H * ell)) / (1 - np.exp(2 * ell))
            assert abs(oracle.lifetime_weight(ell, H) - ref) <= 1e-9 * ref
    assert oracle.lifetime_weight(0.0, 100) == 100


def _brute(cost, cands, fits):
    U, K = cost.shape
    best, arg = np.inf, None
    for ch in itertools.product(range(K), repeat=U):
        if not fits(sum(cands[k] for k in ch)):
            continue
        val = sum(cost[u, k] for u, k in enumerate(ch))
        if val < best:
            best, arg = val, ch
    return best, arg


def _random_costs(rng, U, cands):
    d = np.sort(np.exp(rng.normal(0, 2, (U, len(cands)))), axis=1)[:, ::-1]   # decreasing in b
    return d * np.exp(rng.normal(0, 1, (U, 1)))


@pytest.mark.parametrize("cands", [(4, 6, 8), (2, 4, 6, 8)])
def test_dp_equals_brute_force(oracle, rng, cands):
    for _ in range(25):
        U = int(rng.integers(1, 7))
        cost = _random_costs(rng, U, cands)
        cap = int(rng.integers(min(cands) // 2 * U, max(cands) // 2 * U + 1))
        ch = oracle.allocate_dp(cost, cands, cap)
        best, _ = _brute(cost, cands, lambda bits: bits <= 2 * cap)
        assert ch is not None
        assert sum(cands[k] for k in ch) <= 2 * cap
        assert abs(sum(cost[u, k] for u, k in enumerate(ch)) - best) <= 1e-12 * best
    assert oracle.allocate_dp(np.ones((3, 3)), (4, 6, 8), 5) is None          # 3 units need >= 6


@pytest.mark.parametrize("cands", [(4, 6, 8), (2, 4, 6, 8)])
def test_lagrangian_feasible_and_near_optimal(oracle, rng, cands):
    excess = []
    for _ in range(25):
        U = int(rng.integers(2, 7))
        cost = _random_costs(rng, U, cands)
        budget = int(rng.integers(min(cands) * U, max(cands) * U + 1))
        ch = oracle.allocate_lagrangian(cost, cands, budget)
        best, _ = _brute(cost, cands, lambda bits: bits <= budget)
        val = sum(cost[u, k] for u, k in enumerate(ch))
        assert sum(cands[k] for k in ch) <= budget
        assert val >= best * (1 - 1e-12)
        assert val <= best + np.max(cost[:, 0] - cost[:, -1])
        excess.append(val / best - 1)
    assert np.median(excess) < 0.05
    assert oracle.allocate_lagrangian(np.ones((3, 3)), (4, 6, 8), 11) is None


def test_lagrangian_uses_whole_budget_when_everything_fits(oracle, rng):
    cost = _random_costs(rng, 5, (2, 4, 6, 8))
    ch = oracle.allocate_lagrangian(cost, (2, 4, 6, 8), 40)
    assert all(k == 3 for k in ch)


def test_head_pivots_rank_residual_risk(oracle, rng):
    cands = (4, 6, 8)
    U, nominal, n_piv = 6, 6, 2
    dist = np.concatenate([_random_costs(rng, U, cands), 1e-9 * np.ones((U, 1))], axis=1)
    L = np.exp(rng.normal(0, 1, U))
    piv = oracle.select_pivots(HEAD, cands, nominal, L, dist, n_piv)
    _, arg = _brute(L[:, None] * dist[:, :3], cands, lambda bits: bits <= nominal * U)
    risk = np.array([L[u] * dist[u, k] for u, k in enumerate(arg)])
    assert set(np.flatnonzero(piv)) == set(np.argsort(-risk, kind="stable")[:n_piv])
    bits = oracle.allocate(HEAD, cands, nominal, L, dist, piv)
    assert np.all(bits[piv == 1] == 16)
    # pivots are 8-bit replacements against the nominal budget
    assert np.sum(bits[piv == 0]) + 8 * n_piv <= nominal * U


@pytest.mark.parametrize("fp16_share", [0.0, 0.95])
def test_row_pivots_rank_fp16_reduction(oracle, rng, fp16_share):
    """Row pivots go to the largest L_u (d_u(nominal) - d_u(FP16)); with the FP16
    distortion a large share of d_u(nominal) the ranking differs from L d alone."""
    cands = (2, 4, 6, 8)
    U = 40
    d = _random_costs(rng, U, cands)
    L = np.exp(rng.normal(0, 1, U))
    d16 = np.exp(rng.normal(-12, 1, U))
    plain_top = np.argsort(-(L * d[:, 1]), kind="stable")[:5]
    d16[plain_top] += fp16_share * d[plain_top, 1]      # FP16 barely helps these rows
    dist = np.concatenate([d, d16[:, None]], axis=1)
    piv = oracle.select_pivots(ROW, cands, 4, L, dist, 5)
    risk = L * (dist[:, 1] - dist[:, 4])
    assert set(np.flatnonzero(piv)) == set(np.argsort(-risk, kind="stable")[:5])
    if fp16_share > 0:
        assert set(np.flatnonzero(piv)) != set(plain_top)
    bits = oracle.allocate(ROW, cands, 4, L, dist, piv)
    assert np.sum(bits[piv == 0]) + 8 * 5 <= 4 * U


def _paper_plan(oracle, rng, g):
    n_units = g["layers"] * g["heads"] * (1 if g["unit"] == "head" else D)
    unit = HEAD if g["unit"] == "head" else ROW
    cands = tuple(g["candidates"])
    dist = np.concatenate([_random_costs(rng, n_units, cands),
                           np.exp(rng.normal(-14, 1, (n_units, 1)))], axis=1)
    L = np.exp(rng.normal(3, 1, n_units))
    piv = oracle.select_pivots(unit, cands, g["nominal"], L, dist, g["pivots"])
    bits = oracle.allocate(unit, cands, g["nominal"], L, dist, piv)
    off, nb, stride = oracle.layout(unit, g["layers"], g["heads"], bits)
    return unit, bits, off, nb, stride


def test_qwen_at6_packed_bytes(oracle, rng):
    """App. F.1: 29,999,104 B per request; App. F.3: 30,015,488 B with pivot scale
    slots; Eq. compact_qwen: 6.3611 bits/value."""
    g = GOLD["qwen_at6"]
    unit, bits, off, nb, stride = _paper_plan(oracle, rng, g)
    assert int(np.sum(bits == 16)) == g["pivots"]
    total = int(np.sum(nb))
    assert total == g["packed_bytes"] == stride
    assert total + 512 * g["pivots"] == g["packed_bytes_with_pivot_scale_slots"]
    N = g["layers"] * g["heads"] * D * D
    assert 4 * N == g["fp32_bytes"]
    assert round((total + 512 * g["pivots"]) * 8 / N, 4) == g["compact_bits"]
    assert np.all(off % 16 == 0) and np.all(np.diff(off.astype(np.int64)) == nb[:-1])


@pytest.mark.parametrize("key", ["kda_at6", "kda_at4"])
def test_kda_packed_bytes(oracle, rng, key):
    """App. D: KDA @6 = 7.875 MiB (6.30 bits/value), @4 = 5.375 MiB (4.30)."""
    g = GOLD[key]
    unit, bits, off, nb, stride = _paper_plan(oracle, rng, g)
    total = int(np.sum(nb))
    assert total == g["mib"] * 2 ** 20
    N = g["layers"] * g["heads"] * D * D
    assert round(total * 8 / N, 2) == g["compact_bits"]
    if "fp32_mib" in g:
        assert 4 * N == g["fp32_mib"] * 2 ** 20
    assert stride % 256 == 0 and stride >= total


def _pick(cost, cands, lam):
    """argmin_k cost[u][k] + lam cands[k] per unit, ties to the narrower code
    (the relaxed problem of App. C.2, written out with numpy)."""
    b = np.asarray(cands, np.float64)
    order = np.argsort(b, kind="stable")
    val = cost[:, order] + lam * b[order]
    return order[np.argmin(val, axis=1)]


@pytest.mark.parametrize("cands", [(4, 6, 8), (2, 4, 6, 8)])
def test_lagrangian_multiplier_is_the_budget_threshold(oracle, rng, cands):
    """The shared multiplier is the smallest lambda whose relaxed choices fit:
    they fit at lambda, and just below it they do not (0 when everything fits)."""
    c = np.asarray(cands)
    for _ in range(40):
        U = int(rng.integers(2, 9))
        cost = _random_costs(rng, U, cands)
        budget = int(rng.integers(min(cands) * U, max(cands) * U + 1))
        lam = oracle.lagrangian_multiplier(cost, cands, budget)
        assert lam is not None and lam >= 0.0
        assert c[_pick(cost, cands, lam)].sum() <= budget
        if lam > 0.0:
            assert c[_pick(cost, cands, lam * (1 - 1e-9))].sum() > budget
        else:
            assert c[_pick(cost, cands, 0.0)].sum() <= budget
    assert oracle.lagrangian_multiplier(np.ones((3, 3)), (4, 6, 8), 11) is None


@pytest.mark.parametrize("cands", [(4, 6, 8), (2, 4, 6, 8)])
def test_repair_leaves_no_fitting_upgrade(oracle, rng, cands):
    """The discrete repair upgrades while an upgrade with non-negative gain still
    fits the remaining budget; afterwards none does."""
    for _ in range(40):
        U = int(rng.integers(2, 9))
        cost = _random_costs(rng, U, cands)
        budget = int(rng.integers(min(cands) * U, max(cands) * U + 1))
        ch = oracle.allocate_lagrangian(cost, cands, budget)
        slack = budget - sum(cands[k] for k in ch)
        assert slack >= 0
        for u, cur in enumerate(ch):
            for k, b in enumerate(cands):
                db = b - cands[cur]
                if 0 < db <= slack:
                    assert cost[u, cur] - cost[u, k] < 0, (u, cur, k, slack)


def test_layout_offsets_and_stride(oracle):
    """Head segments follow one another in (layer, head) order, each as long as
    its head page; the slot stride is their sum rounded up to 256 bytes. The row
    widths make one head page 128 bytes past a multiple of 256."""
    rb = np.full(D, 4, np.int8)
    rb[:4] = 6                                      # sum of widths = 520 = 8 (mod 16)
    rb2 = np.full(D, 8, np.int8)
    bits = np.concatenate([rb, rb2, rb])
    off, nb, stride = oracle.layout(ROW, 3, 1, bits)
    sizes = [512 + 16 * int(r.astype(int).sum()) for r in (rb, rb2, rb)]
    assert list(nb) == sizes
    assert list(off) == [0, sizes[0], sizes[0] + sizes[1]]
    assert sizes[0] % 256 == 128
    assert stride % 256 == 0 and 0 <= stride - sum(sizes) < 256
    assert oracle.layout(ROW, 1, 1, rb)[2] == 8960


def test_dp_keeps_the_wider_code_on_ties(oracle):
    """The DP's tie rule (a reading; the paper fixes none): among choices of equal
    cost it keeps the wider code, so equal costs with room for every unit at the
    widest candidate give the widest."""
    for cands in ((4, 6, 8), (2, 4, 6, 8)):
        ch = oracle.allocate_dp(np.zeros((5, len(cands))), cands, max(cands) // 2 * 5)
        assert all(cands[k] == max(cands) for k in ch)
