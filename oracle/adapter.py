"""Oracle: the FrameFT adapter update and its gradients, dense fp64.

Test infrastructure only (see ``oracle/__init__``).

Notation of Sec. 3.1: W in R^{m x n} (out x in), P_m = Phi_out (m x K_m),
P_n = Phi_in (n x K_n), C in R^{K_m x K_n}, s = alpha / sqrt(mn) and

    dW = s * P_m C P_n^T                      (update equation, Alg. 1 step 5)
    W' = W + dW                               (Alg. 1 step 6)

Activations are row-major (one token per row): X is N x n, Y and dY are N x m,
so the layer computes Y = X W'^T.  Everything here forms dW explicitly with
numpy matmuls in fp64 -- no blocking, fusion or reordering.
"""
from __future__ import annotations

import numpy as np


def dense_C(rows: int, cols: int, row: np.ndarray, col: np.ndarray, val: np.ndarray) -> np.ndarray:
    """Dense coefficient matrix from its support (Alg. 1 step 4, 'rearrange')."""
    C = np.zeros((rows, cols), dtype=np.float64)
    C[np.asarray(row, dtype=np.int64), np.asarray(col, dtype=np.int64)] = np.asarray(val, dtype=np.float64)
    return C


def delta_w(phi_out: np.ndarray, C: np.ndarray, phi_in: np.ndarray, scale: float) -> np.ndarray:
    """dW = s P_m C P_n^T (Sec. 3.1 update equation; Alg. 1 step 5)."""
    return scale * (phi_out @ C @ phi_in.T)


def forward(X, Y_in, phi_in, phi_out, C, scale):
    """Y_out = Y_in + X dW^T: the adapter's contribution accumulated onto the
    frozen layer's output (Alg. 1 step 6 applied to a batch of rows)."""
    return np.asarray(Y_in, dtype=np.float64) + np.asarray(X, dtype=np.float64) @ delta_w(phi_out, C, phi_in, scale).T


def backward_dx(dY, dX_in, phi_in, phi_out, C, scale):
    """dX_out = dX_in + dY dW: gradient of Y = X dW^T with respect to X."""
    return np.asarray(dX_in, dtype=np.float64) + np.asarray(dY, dtype=np.float64) @ delta_w(phi_out, C, phi_in, scale)


def grad_coeff_full(X, dY, phi_in, phi_out, scale):
    """Dense coefficient gradient s P_m^T grad_W P_n with grad_W = dY^T X
    (Lemma 1 proof, Appendix A: grad f(C) = P_m^T grad f(W) P_n; the factor s
    comes from the scaled update equation)."""
    gW = np.asarray(dY, dtype=np.float64).T @ np.asarray(X, dtype=np.float64)
    return scale * (phi_out.T @ gW @ phi_in)


def grad_coeff(X, dY, phi_in, phi_out, scale, row, col):
    """The coefficient gradient sampled on the support of C (only the support
    entries are trainable, Sec. 3.3)."""
    G = grad_coeff_full(X, dY, phi_in, phi_out, scale)
    return G[np.asarray(row, dtype=np.int64), np.asarray(col, dtype=np.int64)]


def merge(W0, C_list, phi_in, phi_out, scale):
    """W_t = W0 + dW(C_t) for every tenant t (Alg. 1 step 6, one adapter per
    tenant over a shared backbone -- Sec. 3.4 'Storage efficiency')."""
    W0 = np.asarray(W0, dtype=np.float64)
    return np.stack([W0 + delta_w(phi_out, C, phi_in, scale) for C in C_list])
