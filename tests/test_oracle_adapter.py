"""Pins of the oracle's adapter arithmetic: brute force, linearity, isometry,
adjoint identities, finite differences and the merge identity."""
import itertools

import numpy as np
import pytest

from oracle import adapter, frames, support


def _setup(m, n, k_m, k_n, rho_m, rho_n, nnz, seed=3, parseval=True):
    Pm = frames.real_frame(m, k_m, rho_m, parseval)
    Pn = frames.real_frame(n, k_n, rho_n, parseval)
    Km, Kn = Pm.shape[1], Pn.shape[1]
    row, col, _, _ = support.sample_support(Km, Kn, nnz, seed)
    rng = np.random.default_rng(seed)
    val = rng.standard_normal(nnz)
    return Pm, Pn, row, col, val


# (m, n, k_m, k_n, rho_m, rho_n): square and non-square, k*rho = d and redundant frames
SHAPES = [(4, 4, 2, 2, 2, 2), (8, 8, 4, 4, 2, 2), (8, 8, 2, 2, 4, 4), (12, 12, 6, 6, 2, 2),
          (12, 12, 3, 3, 4, 4), (8, 12, 2, 2, 4, 6), (12, 8, 6, 4, 2, 2), (22, 22, 6, 6, 6, 6)]


@pytest.mark.parametrize("shape", SHAPES)
def test_delta_w_brute_force(shape):
    m, n, km, kn, rm, rn = shape
    Pm, Pn, row, col, val = _setup(m, n, km, kn, rm, rn, nnz=min(7, km * rm * kn * rn))
    Km, Kn = Pm.shape[1], Pn.shape[1]
    s = 0.37
    C = adapter.dense_C(Km, Kn, row, col, val)
    got = adapter.delta_w(Pm, C, Pn, s)
    want = np.zeros((m, n))
    for i, j in itertools.product(range(m), range(n)):
        acc = 0.0
        for a, b in itertools.product(range(Km), range(Kn)):
            acc += Pm[i, a] * C[a, b] * Pn[j, b]
        want[i, j] = s * acc
    np.testing.assert_allclose(got, want, atol=1e-13)


@pytest.mark.parametrize("shape", SHAPES[:6])
def test_forward_dx_dc_brute_force(shape):
    m, n, km, kn, rm, rn = shape
    Pm, Pn, row, col, val = _setup(m, n, km, kn, rm, rn, nnz=min(5, km * rm * kn * rn))
    Km, Kn = Pm.shape[1], Pn.shape[1]
    s = 1.7
    C = adapter.dense_C(Km, Kn, row, col, val)
    rng = np.random.default_rng(11)
    N = 3
    X, dY = rng.standard_normal((N, n)), rng.standard_normal((N, m))
    Y0, dX0 = rng.standard_normal((N, m)), rng.standard_normal((N, n))
    Y = adapter.forward(X, Y0, Pn, Pm, C, s)
    dX = adapter.backward_dx(dY, dX0, Pn, Pm, C, s)
    dC = adapter.grad_coeff(X, dY, Pn, Pm, s, row, col)
    for t in range(N):
        for i in range(m):           # Y[t,i] = Y0 + sum_j X[t,j] dW[i,j]
            acc = sum(X[t, j] * s * Pm[i, a] * C[a, b] * Pn[j, b]
                      for j in range(n) for a in range(Km) for b in range(Kn) if C[a, b] != 0)
            assert abs(Y[t, i] - Y0[t, i] - acc) < 1e-12
        for j in range(n):           # dX[t,j] = dX0 + sum_i dY[t,i] dW[i,j]
            acc = sum(dY[t, i] * s * Pm[i, a] * C[a, b] * Pn[j, b]
                      for i in range(m) for a in range(Km) for b in range(Kn) if C[a, b] != 0)
            assert abs(dX[t, j] - dX0[t, j] - acc) < 1e-12
    for q, (a, b) in enumerate(zip(row, col)):   # dC_q = s sum_t sum_ij dY[t,i] Pm[i,a] X[t,j] Pn[j,b]
        acc = sum(dY[t, i] * Pm[i, a] * X[t, j] * Pn[j, b] for t in range(N) for i in range(m) for j in range(n))
        assert abs(dC[q] - s * acc) < 1e-12


def test_linearity_in_C():
    Pm, Pn, row, col, val = _setup(64, 48, 8, 8, 8, 6, nnz=40)
    Km, Kn = Pm.shape[1], Pn.shape[1]
    rng = np.random.default_rng(5)
    C1 = adapter.dense_C(Km, Kn, row, col, rng.standard_normal(40))
    C2 = adapter.dense_C(Km, Kn, row, col, rng.standard_normal(40))
    a, b = 0.7, -2.3
    lhs = adapter.delta_w(Pm, a * C1 + b * C2, Pn, 0.5)
    rhs = a * adapter.delta_w(Pm, C1, Pn, 0.5) + b * adapter.delta_w(Pm, C2, Pn, 0.5)
    np.testing.assert_allclose(lhs, rhs, atol=1e-13)


@pytest.mark.parametrize("m,n", [(256, 256), (64, 96)])
def test_isometry_for_orthonormal_frames(m, n):
    # k*rho = d and Parseval: P is orthogonal, so ||dW||_F = s ||C||_F (equality
    # case of the bound ||W1 - W2||_F <= sqrt(B_m B_n) ||C1 - C2||_F, Lemma 1 proof)
    Pm, Pn, row, col, val = _setup(m, n, 16, 16, m // 16, n // 16, nnz=100)
    C = adapter.dense_C(Pm.shape[1], Pn.shape[1], row, col, val)
    s = 0.25
    assert np.isclose(np.linalg.norm(adapter.delta_w(Pm, C, Pn, s)), s * np.linalg.norm(C), rtol=1e-13)


def test_lipschitz_bound_for_redundant_frame():
    # non-Parseval redundant frame: ||dW||_F <= sqrt(B_m B_n) s ||C||_F with B = 18/11
    Pm, Pn, row, col, val = _setup(22, 22, 6, 6, 6, 6, nnz=60, parseval=False)
    C = adapter.dense_C(36, 36, row, col, val)
    B = 18.0 / 11.0
    assert np.linalg.norm(adapter.delta_w(Pm, C, Pn, 1.0)) <= B * np.linalg.norm(C) * (1 + 1e-12)


@pytest.mark.parametrize("shape", [(64, 96, 8, 8, 8, 12), (22, 22, 6, 6, 6, 6), (96, 64, 16, 16, 6, 4)])
def test_adjoint_identities(shape):
    m, n, km, kn, rm, rn = shape
    Pm, Pn, row, col, val = _setup(m, n, km, kn, rm, rn, nnz=50)
    Km, Kn = Pm.shape[1], Pn.shape[1]
    s = 0.8
    C = adapter.dense_C(Km, Kn, row, col, val)
    rng = np.random.default_rng(9)
    X, dY = rng.standard_normal((17, n)), rng.standard_normal((17, m))
    Z = np.zeros((17, m))
    fwd = adapter.forward(X, Z, Pn, Pm, C, s)
    bwd = adapter.backward_dx(dY, np.zeros((17, n)), Pn, Pm, C, s)
    dC = adapter.grad_coeff(X, dY, Pn, Pm, s, row, col)
    a = np.sum(dY * fwd)
    b = np.dot(dC, val)
    c = np.sum(bwd * X)
    assert np.isclose(a, b, rtol=1e-12) and np.isclose(a, c, rtol=1e-12)


def test_finite_differences():
    Pm, Pn, row, col, val = _setup(32, 48, 4, 4, 8, 12, nnz=30)
    Km, Kn = Pm.shape[1], Pn.shape[1]
    s = 1.3
    rng = np.random.default_rng(12)
    X, G = rng.standard_normal((6, 48)), rng.standard_normal((6, 32))

    def loss(v, Xv):
        C = adapter.dense_C(Km, Kn, row, col, v)
        return np.sum(G * adapter.forward(Xv, np.zeros((6, 32)), Pn, Pm, C, s))

    dC = adapter.grad_coeff(X, G, Pn, Pm, s, row, col)
    dX = adapter.backward_dx(G, np.zeros_like(X), Pn, Pm, adapter.dense_C(Km, Kn, row, col, val), s)
    h = 1e-6
    for q in range(0, 30, 7):
        e = np.zeros(30)
        e[q] = h
        fd = (loss(val + e, X) - loss(val - e, X)) / (2 * h)
        assert abs(fd - dC[q]) < 1e-7 * max(1.0, abs(dC[q]))
    for (t, j) in [(0, 0), (3, 17), (5, 47)]:
        E = np.zeros_like(X)
        E[t, j] = h
        fd = (loss(val, X + E) - loss(val, X - E)) / (2 * h)
        assert abs(fd - dX[t, j]) < 1e-7 * max(1.0, abs(dX[t, j]))


def test_merge_matches_forward():
    Pm, Pn, row, col, _ = _setup(64, 96, 8, 8, 8, 12, nnz=25)
    Km, Kn = Pm.shape[1], Pn.shape[1]
    rng = np.random.default_rng(4)
    W0 = 0.02 * rng.standard_normal((64, 96))
    vals = [rng.standard_normal(25) for _ in range(3)]
    Cs = [adapter.dense_C(Km, Kn, row, col, v) for v in vals]
    s = 0.4
    W = adapter.merge(W0, Cs, Pn, Pm, s)
    X = rng.standard_normal((5, 96))
    for t in range(3):
        np.testing.assert_allclose(X @ (W[t] - W0).T,
                                   adapter.forward(X, np.zeros((5, 64)), Pn, Pm, Cs[t], s), atol=1e-13)
