"""Oracle: random sparse support of the coefficient matrix C (pure Python).

Test infrastructure only (see ``oracle/__init__``).

Sec. 3.3: a small random subset of the entries of C is non-zero, and the same
index set is shared by every layer of a shape.  The paper does not fix a
generator, so the support is drawn from a splitmix64 stream (S. Vigna's
published generator; state += 0x9e3779b97f4a7c15, then two xor-shift-multiply
rounds) with these rules, which the C library follows bit for bit:

* ``uniform_int(R)`` = ((next() >> 11) * R) >> 53 (exact 128-bit product).
* ``uniform_01()``   = (next() >> 11) * 2^-53.
* UNIFORM   (mode 0): one draw ``p = uniform_int(rows*cols)``; (a, b) = divmod(p, cols).
* ZIPF_ROWS (mode 1): a = smallest r with cdf[r] > uniform_01() * cdf[rows-1],
  cdf[r] = sum_{i<=r} (i+1)^-s summed left to right in fp64; then b = uniform_int(cols).
* BLOCKDIAG (mode 2): block i = uniform_int(k); a = i*rows/k + uniform_int(rows/k),
  b = i*cols/k + uniform_int(cols/k) -- the k diagonal blocks C_{l,i} of Sec. 3.1.
* A drawn position already in the set is discarded and drawing continues
  until nnz distinct positions are held.

Output: the positions sorted row-major, the CSR row pointer over a, and the
permutation that orders the entries by (b, a).
"""
from __future__ import annotations

import bisect

import numpy as np

MASK64 = (1 << 64) - 1
GOLDEN = 0x9E3779B97F4A7C15

UNIFORM, ZIPF_ROWS, BLOCKDIAG = 0, 1, 2


class SplitMix64:
    def __init__(self, seed: int):
        self.state = seed & MASK64

    def next(self) -> int:
        self.state = (self.state + GOLDEN) & MASK64
        z = self.state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
        return z ^ (z >> 31)

    def uniform_int(self, r: int) -> int:
        return ((self.next() >> 11) * r) >> 53

    def uniform_01(self) -> float:
        return (self.next() >> 11) * (1.0 / 9007199254740992.0)


def zipf_cdf(rows: int, s: float) -> list[float]:
    cdf, acc = [], 0.0
    for r in range(1, rows + 1):
        acc += float(r) ** (-s)
        cdf.append(acc)
    return cdf


def sample_support(rows: int, cols: int, nnz: int, seed: int, mode: int = UNIFORM,
                   zipf_s: float = 1.1, k: int = 1):
    """Distinct support positions of C (rows x cols), sorted row-major.

    Returns (row int32[nnz], col int32[nnz], csr_rowptr int64[rows+1],
    csc_perm int32[nnz]).
    """
    if nnz < 0 or nnz > rows * cols:
        raise ValueError("nnz out of range")
    rng = SplitMix64(seed)
    chosen: set[tuple[int, int]] = set()
    cdf = zipf_cdf(rows, zipf_s) if mode == ZIPF_ROWS else None
    if mode == BLOCKDIAG:
        if k < 1 or rows % k or cols % k:
            raise ValueError("BLOCKDIAG needs k dividing rows and cols")
        if nnz > k * (rows // k) * (cols // k):
            raise ValueError("nnz exceeds the block-diagonal capacity")
    while len(chosen) < nnz:
        if mode == UNIFORM:
            p = rng.uniform_int(rows * cols)
            a, b = divmod(p, cols)
        elif mode == ZIPF_ROWS:
            u = rng.uniform_01() * cdf[-1]
            a = bisect.bisect_right(cdf, u)
            if a >= rows:
                a = rows - 1
            b = rng.uniform_int(cols)
        elif mode == BLOCKDIAG:
            i = rng.uniform_int(k)
            rb, cb = rows // k, cols // k
            a = i * rb + rng.uniform_int(rb)
            b = i * cb + rng.uniform_int(cb)
        else:
            raise ValueError("unknown support mode")
        chosen.add((a, b))
    pos = sorted(chosen)
    row = np.array([a for a, _ in pos], dtype=np.int32)
    col = np.array([b for _, b in pos], dtype=np.int32)
    rowptr = np.zeros(rows + 1, dtype=np.int64)
    for a in row:
        rowptr[a + 1] += 1
    rowptr = np.cumsum(rowptr)
    perm = sorted(range(nnz), key=lambda q: (int(col[q]), int(row[q])))
    return row, col, rowptr.astype(np.int64), np.asarray(perm, dtype=np.int32)
