"""Pins of the oracle's FP32-state gated Delta rule (Sec. 2.1, Prop. 1, App. A, App. B).

Each check compares the oracle with a fact the paper fixes independently of
the oracle's own loops: the second algebraic form of Eq. delta_update, the
directional contraction of Eq. self_correction, the bound ||A_t||_2 <= 1 of
Prop. 1, and the readout identity ||E_i^T g_t||^2 = g_{t,i}^2 (App. B.3).
"""
import json
import os

import numpy as np
import pytest

D = 128


def _inputs(rng, per_row=False, knorm=1.0):
    q = rng.standard_normal(D).astype(np.float32)
    k = rng.standard_normal(D)
    k = (knorm * k / np.linalg.norm(k)).astype(np.float32)
    v = rng.standard_normal(D).astype(np.float32)
    beta = np.float32(rng.uniform(0.05, 0.95))
    gate = (rng.uniform(0.8, 0.999, size=D) if per_row else
            np.array([rng.uniform(0.85, 0.999)])).astype(np.float32)
    return q, k, v, beta, gate


@pytest.mark.parametrize("per_row", [False, True])
def test_step_matches_affine_form(oracle, rng, per_row):
    """S_t = (I - beta k k^T) D S + beta k v^T  (right-hand form of Eq. delta_update)."""
    S = (rng.standard_normal((D, D)) * np.exp(rng.normal(size=(D, 1)))).astype(np.float32)
    q, k, v, beta, gate = _inputs(rng, per_row)
    S1, y = oracle.delta_step(S, q, k, v, beta, gate)
    Dm = np.diag(np.broadcast_to(gate.astype(np.float64), (D,)))
    kk = k.astype(np.float64)
    A = (np.eye(D) - float(beta) * np.outer(kk, kk)) @ Dm
    ref = A @ S.astype(np.float64) + float(beta) * np.outer(kk, v.astype(np.float64))
    scale = np.abs(ref).max()
    assert np.abs(S1 - ref).max() <= 4e-7 * scale
    # readout from the updated state, y = S_t^T q
    yref = S1.astype(np.float64).T @ q.astype(np.float64)
    assert np.abs(y - yref).max() <= 1e-6 * np.abs(yref).max()


def _transition(oracle, q, k, beta, gate):
    """A_t as the oracle applies it: one step of S = I with v = 0 gives A_t I."""
    S1, _ = oracle.delta_step(np.eye(D, dtype=np.float32), q, k, np.zeros(D, np.float32), beta, gate)
    return S1.astype(np.float64)


@pytest.mark.parametrize("per_row", [False, True])
def test_transition_is_non_expansive(oracle, rng, per_row):
    """Prop. 1: ||k|| <= 1, 0 <= beta <= 1, 0 <= D <= I  =>  ||A_t||_2 <= ||D_t||_2 <= 1."""
    for _ in range(3):
        q, k, v, beta, gate = _inputs(rng, per_row, knorm=rng.uniform(0.3, 1.0))
        A = _transition(oracle, q, k, beta, gate)
        smax = np.linalg.svd(A, compute_uv=False)[0]
        assert smax <= float(np.max(gate)) * (1 + 1e-6) <= 1.0 + 1e-6


def test_directional_contraction(oracle, rng):
    """Eq. self_correction: ||a(I - b k k^T)E||_F^2 = a^2[||E||^2 - b(2 - b||k||^2)||k^T E||^2]."""
    for knorm in (1.0, 0.7):
        q, k, v, beta, gate = _inputs(rng, False, knorm)
        E = rng.standard_normal((D, D)).astype(np.float32)
        E1, _ = oracle.delta_step(E, q, k, np.zeros(D, np.float32), beta, gate)   # v = 0: E1 = A E
        a, b = float(gate[0]), float(beta)
        k64, E64 = k.astype(np.float64), E.astype(np.float64)
        rhs = a * a * (np.sum(E64 ** 2) - b * (2 - b * k64 @ k64) * np.sum((k64 @ E64) ** 2))
        lhs = np.sum(E1.astype(np.float64) ** 2)
        assert abs(lhs - rhs) <= 1e-6 * rhs


@pytest.mark.parametrize("per_row", [False, True])
def test_exact_read_error_is_only_decayed(oracle, rng, per_row):
    """App. B.1: with the residual reading the reference state, the path's error
    evolves as E_t = D_t E_{t-1}, while the native step gives (I - beta k k^T) D E."""
    S_ref = (rng.standard_normal((D, D)) * np.exp(rng.normal(size=(D, 1)))).astype(np.float32)
    E = (1e-2 * rng.standard_normal((D, D)) * np.abs(S_ref).max()).astype(np.float32)
    S = (S_ref.astype(np.float64) + E).astype(np.float32)
    E = S.astype(np.float64) - S_ref.astype(np.float64)
    q, k, v, beta, gate = _inputs(rng, per_row)
    # reference trajectory: the plain step of S_ref, written out here in fp64
    g = np.broadcast_to(gate.astype(np.float64), (D,))
    k64, b = k.astype(np.float64), float(beta)
    P_ref = g[:, None] * S_ref.astype(np.float64)
    ref1 = P_ref + b * np.outer(k64, v.astype(np.float64) - k64 @ P_ref)
    S1, y = oracle.delta_step_read(S, S_ref, q, k, v, beta, gate)
    scale = np.abs(ref1).max()
    assert np.abs((S1 - ref1) - g[:, None] * E).max() <= 1e-6 * scale
    assert np.abs(y - S1.astype(np.float64).T @ q.astype(np.float64)).max() <= 1e-6 * np.abs(y).max()
    # the native step of the same perturbed state removes the k-direction of D E
    N1, _ = oracle.delta_step(S, q, k, v, beta, gate)
    DE = g[:, None] * E
    assert np.abs((N1 - ref1) - (DE - b * np.outer(k64, k64 @ DE))).max() <= 1e-6 * scale
    # and with S = S_ref the two steps coincide
    X1, _ = oracle.delta_step_read(S_ref, S_ref, q, k, v, beta, gate)
    R1, _ = oracle.delta_step(S_ref, q, k, v, beta, gate)
    assert np.abs(X1 - R1).max() <= 4e-7 * scale


def test_exact_read_batch_matches_single_steps(oracle, rng):
    n, Hk, Hv = 2, 1, 2
    S = rng.standard_normal((n, Hv, D, D)).astype(np.float32)
    S_ref = (S + 0.1 * rng.standard_normal(S.shape)).astype(np.float32)
    q = rng.standard_normal((n, Hk, D)).astype(np.float32)
    k = rng.standard_normal((n, Hk, D)).astype(np.float32) / np.sqrt(D)
    v = rng.standard_normal((n, Hv, D)).astype(np.float32)
    beta = rng.uniform(0.1, 0.9, (n, Hv)).astype(np.float32)
    gate = rng.uniform(0.8, 1.0, (n, Hv, D)).astype(np.float32)
    Sb = S.copy()
    y = oracle.delta_batch_read(Sb, S_ref, q, k, v, beta, gate)
    for b in range(n):
        for h in range(Hv):
            s1, y1 = oracle.delta_step_read(S[b, h], S_ref[b, h], q[b, 0], k[b, 0], v[b, h],
                                            beta[b, h], gate[b, h])
            assert np.array_equal(Sb[b, h], s1) and np.array_equal(y[b, h], y1)


@pytest.mark.parametrize("per_row", [False, True])
def test_row_impact_closed_form_and_readout_identity(oracle, rng, per_row):
    """g_t = A_t^T q_t (Sec. 4.1; Eq. kda_sensitivity) and the App. B.3 identity:
    a unit-norm perturbation confined to key row i changes the next readout by
    exactly g_{t,i}^2 in squared norm."""
    golden = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "storage.json")))
    tol = golden["readout_identity_rel_err"]["value"] * 20      # fp32 state vs the paper's check
    q, k, v, beta, gate = _inputs(rng, per_row)
    g = oracle.row_impact(q, k, beta, gate)
    g_dense = oracle.row_impact(q, k, beta, gate, dense=True)
    A = _transition(oracle, q, k, beta, gate)
    g_from_step = A.T @ q.astype(np.float64)
    assert np.allclose(g, g_dense, rtol=1e-12, atol=1e-12)
    assert np.allclose(g, g_from_step, rtol=1e-5, atol=1e-6 * np.abs(g).max())
    for i in rng.choice(D, size=6, replace=False):
        e = rng.standard_normal(D)
        E = np.zeros((D, D), np.float32)
        E[i] = (e / np.linalg.norm(e)).astype(np.float32)
        _, dy = oracle.delta_step(E, q, k, np.zeros(D, np.float32), beta, gate)   # y(E) = (A E)^T q
        err = np.sum(dy.astype(np.float64) ** 2)
        assert abs(err - g[i] ** 2) <= tol * max(g[i] ** 2, 1e-3 * np.max(g ** 2)) + 1e-9


def test_batch_driver_matches_single_steps(oracle, rng):
    n, Hk, Hv = 2, 2, 4
    S = rng.standard_normal((n, Hv, D, D)).astype(np.float32)
    q = rng.standard_normal((n, Hk, D)).astype(np.float32)
    k = rng.standard_normal((n, Hk, D)).astype(np.float32)
    k /= np.linalg.norm(k, axis=-1, keepdims=True)
    v = rng.standard_normal((n, Hv, D)).astype(np.float32)
    beta = rng.uniform(0, 1, (n, Hv)).astype(np.float32)
    gate = rng.uniform(0.9, 1, (n, Hv)).astype(np.float32)
    S0 = S.copy()
    y = oracle.delta_batch(S, q, k, v, beta, gate)
    for b in range(n):
        for h in range(Hv):
            s1, y1 = oracle.delta_step(S0[b, h], q[b, h // 2], k[b, h // 2], v[b, h], beta[b, h],
                                       gate[b, h])
            assert np.array_equal(s1, S[b, h]) and np.array_equal(y1, y[b, h])
