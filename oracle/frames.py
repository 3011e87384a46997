"""Oracle: tight fusion frame construction (fp64, numpy).

Test infrastructure only (see ``oracle/__init__``).

Construction of a (k, rho, d) uniform tight fusion frame, following the three
steps of Sec. 3.2 and the appendix walk-through of the (6,3,11) example:

1. Spectral Tetris: a unit-norm tight frame of d_c vectors in C^{rho_c},
   stored as the rho_c x d_c matrix F (columns = frame vectors), rows
   orthogonal with squared norm d_c / rho_c.  Greedy rule: fill a row with
   ones while the norm still to place is >= 1, then close it with the 2x2
   block T(x) (appendix, definition of T(x)) that spills 2 - x onto the next
   row.
2. Modulation: for subspace index k_i in 0..k-1 the rows of F are multiplied
   entrywise by w_{k_i} = (omega^{k_i j})_j, omega = exp(2 pi i / k)
   (appendix, "Modulation").  Subspace k_i is spanned by the rho_c modulated
   rows.
3. Realification: the entrywise map x + iy -> [[x, -y], [y, x]] applied to the
   matrix whose rows are the frame vectors (appendix, first paragraph of the
   Spectral Tetris subsection).  Complex row q becomes real rows 2q, 2q+1;
   complex coordinate j becomes real coordinates 2j, 2j+1.

The real synthesis matrix P (d x k*rho) has the normalised real frame vectors
as columns, ordered subspace-major as P = [P_1, ..., P_k] (Sec. 3.1):
column c = i*rho + 2r + s for subspace i, F-row r, realified part s.
Every vector is scaled to unit norm (d_c / rho_c -> 1); with ``parseval`` the
whole matrix is further scaled by 1/sqrt(A), A = k*rho/d, so that P P^T = I
(Sec. 3.4 chooses Parseval frames for all experiments).
"""
from __future__ import annotations

from fractions import Fraction
import math

import numpy as np


def spectral_tetris(rho_c: int, d_c: int) -> np.ndarray:
    """Spectral Tetris UNTF F (rho_c x d_c, real entries) -- Sec. 3.2 step (1),
    appendix "Spectral Tetris".

    The norm still to place in a row is tracked exactly as a Fraction.
    Requires d_c >= 2 rho_c (otherwise T blocks of consecutive rows would
    overlap); raises ValueError when the greedy walk does not close.
    """
    if rho_c < 1 or d_c < 1:
        raise ValueError("rho_c and d_c must be positive")
    if d_c < 2 * rho_c:
        raise ValueError("Spectral Tetris needs d_c >= 2*rho_c")
    F = np.zeros((rho_c, d_c), dtype=np.float64)
    row_norm = Fraction(d_c, rho_c)
    col = 0
    spilled = Fraction(0)  # norm already placed in this row by the previous T block
    for r in range(rho_c):
        remaining = row_norm - spilled
        while remaining >= 1:
            if col >= d_c:
                raise ValueError("Spectral Tetris ran out of columns")
            F[r, col] = 1.0
            col += 1
            remaining -= 1
        if remaining > 0:
            if r + 1 >= rho_c or col + 1 >= d_c:
                raise ValueError("Spectral Tetris: T block falls outside F")
            x = remaining
            top = math.sqrt(float(x) / 2.0)           # (1/sqrt2) sqrt(x)
            bot = math.sqrt(float(2 - x) / 2.0)       # (1/sqrt2) sqrt(2-x)
            F[r, col] = top
            F[r, col + 1] = top
            F[r + 1, col] = bot
            F[r + 1, col + 1] = -bot
            col += 2
            spilled = 2 - x
        else:
            spilled = Fraction(0)
    if col != d_c:
        raise ValueError("Spectral Tetris did not use every column")
    return F


def row_supports(F: np.ndarray) -> list[tuple[int, int]]:
    """[first, last] column of the nonzero pattern of each row of F."""
    out = []
    for r in range(F.shape[0]):
        nz = np.nonzero(F[r])[0]
        out.append((int(nz[0]), int(nz[-1])))
    return out


def modulation_feasible(F: np.ndarray, k: int) -> bool:
    """The modulated system is tight when no two columns j != j' that share a
    row of F are congruent mod k (the k-th-root sums vanish for all other
    pairs).  Equivalent to k >= the widest row support of F."""
    return all(last - first + 1 <= k for first, last in row_supports(F))


def modulated_frame(k: int, F: np.ndarray) -> np.ndarray:
    """Complex frame vectors omega^{k_i j} F[r, j] -- appendix "Modulation".

    Returns an array M[k_i, r, j] (k x rho_c x d_c).  The exponent k_i * j is
    reduced mod k in integers before the complex exponential is taken.
    """
    rho_c, d_c = F.shape
    M = np.zeros((k, rho_c, d_c), dtype=np.complex128)
    j = np.arange(d_c)
    for ki in range(k):
        expo = (ki * j) % k
        w = np.exp(2j * np.pi * expo / k)
        M[ki] = F * w[None, :]
    return M


def real_frame(d: int, k: int, rho: int, parseval: bool = True) -> np.ndarray:
    """Dense real synthesis matrix P (d x k*rho) of the (k, rho, d) TFF.

    rho and d are the real dimensions; rho_c = rho/2, d_c = d/2.
    Column c = i*rho + 2r + s holds the realified, unit-norm vector of
    subspace i built from F-row r: s = 0 -> (Re z_j, -Im z_j) on coordinates
    (2j, 2j+1); s = 1 -> (Im z_j, Re z_j).
    """
    if rho % 2 or d % 2 or rho < 2:
        raise ValueError("real frames need even rho >= 2 and even d")
    rho_c, d_c = rho // 2, d // 2
    F = spectral_tetris(rho_c, d_c)
    if not modulation_feasible(F, k):
        raise ValueError("modulation by k-th roots of unity is not tight for this F")
    M = modulated_frame(k, F) / math.sqrt(d_c / rho_c)
    P = np.zeros((d, k * rho), dtype=np.float64)
    for i in range(k):
        for r in range(rho_c):
            z = M[i, r]
            c0 = i * rho + 2 * r
            P[0::2, c0] = z.real
            P[1::2, c0] = -z.imag
            P[0::2, c0 + 1] = z.imag
            P[1::2, c0 + 1] = z.real
    if parseval:
        P /= math.sqrt(frame_bound(d, k, rho))
    return P


def frame_bound(d: int, k: int, rho: int) -> float:
    """Tight frame bound A of the unit-norm construction: sum_i P_i P_i^T = A I
    with A = k*rho/d (trace of the frame operator / d)."""
    return k * rho / d


def structural_pattern(d: int, k: int, rho: int) -> np.ndarray:
    """Boolean d x k*rho pattern: the full realified 2x2 block of every nonzero
    entry of F is stored, including entries whose cosine or sine is exactly 0."""
    rho_c, d_c = rho // 2, d // 2
    F = spectral_tetris(rho_c, d_c)
    pat = np.zeros((d, k * rho), dtype=bool)
    for i in range(k):
        for r in range(rho_c):
            js = np.nonzero(F[r])[0]
            for s in (0, 1):
                c = i * rho + 2 * r + s
                pat[2 * js, c] = True
                pat[2 * js + 1, c] = True
    return pat


def csc_from_dense(P: np.ndarray, pattern: np.ndarray):
    """Compressed sparse columns of P over ``pattern`` (rows ascending)."""
    d, K = P.shape
    colptr = np.zeros(K + 1, dtype=np.int64)
    rows, vals = [], []
    for c in range(K):
        rs = np.nonzero(pattern[:, c])[0]
        rows.extend(rs.tolist())
        vals.extend(P[rs, c].tolist())
        colptr[c + 1] = colptr[c] + len(rs)
    return colptr, np.asarray(rows, dtype=np.int32), np.asarray(vals, dtype=np.float64)


def csr_from_dense(P: np.ndarray, pattern: np.ndarray):
    """Compressed sparse rows of P over ``pattern`` (columns ascending)."""
    d, K = P.shape
    rowptr = np.zeros(d + 1, dtype=np.int64)
    cols, vals = [], []
    for j in range(d):
        cs = np.nonzero(pattern[j, :])[0]
        cols.extend(cs.tolist())
        vals.extend(P[j, cs].tolist())
        rowptr[j + 1] = rowptr[j] + len(cs)
    return rowptr, np.asarray(cols, dtype=np.int32), np.asarray(vals, dtype=np.float64)


def group_table(d: int, k: int, rho: int):
    """Per F-row r: the real coordinate range its vectors live on.

    Returns (row0[r], nrows[r]) with row0 = 2*first, nrows = 2*(last-first+1).
    The columns of group r are {i*rho + 2r + s}.
    """
    F = spectral_tetris(rho // 2, d // 2)
    sup = row_supports(F)
    row0 = np.array([2 * a for a, _ in sup], dtype=np.int32)
    nrows = np.array([2 * (b - a + 1) for a, b in sup], dtype=np.int32)
    return row0, nrows
