"""Pins of the oracle's support sampler: the published splitmix64 stream and
distributional / structural properties of each mode."""
import numpy as np
import pytest

from oracle import support


def test_splitmix64_published_stream():
    # first outputs of splitmix64 seeded with 0 (Vigna's reference generator)
    g = support.SplitMix64(0)
    assert [g.next() for _ in range(3)] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def _check_structure(rows, cols, nnz, out):
    row, col, rowptr, perm = out
    assert len(row) == len(col) == nnz
    assert row.min(initial=0) >= 0 and (nnz == 0 or row.max() < rows)
    assert col.min(initial=0) >= 0 and (nnz == 0 or col.max() < cols)
    keys = row.astype(np.int64) * cols + col
    assert np.all(np.diff(keys) > 0)                       # sorted and distinct
    assert rowptr[0] == 0 and rowptr[-1] == nnz
    for a in range(rows):
        assert np.all(row[rowptr[a]:rowptr[a + 1]] == a)
    ck = col.astype(np.int64)[perm] * rows + row[perm]
    assert np.all(np.diff(ck) > 0)                         # perm orders by (col, row)
    assert sorted(perm.tolist()) == list(range(nnz))


@pytest.mark.parametrize("rows,cols,nnz,mode", [(256, 256, 128, 0), (768, 768, 1000, 0), (64, 32, 2048, 0),
                                                (4096, 1024, 3000, 1), (96, 96, 500, 2), (10, 10, 0, 0)])
def test_structure(rows, cols, nnz, mode):
    out = support.sample_support(rows, cols, nnz, seed=1, mode=mode, k=16 if mode == 2 else 1)
    _check_structure(rows, cols, nnz, out)


def test_full_support():
    row, col, _, _ = support.sample_support(6, 5, 30, seed=2)
    assert len(set(zip(row.tolist(), col.tolist()))) == 30


def test_blockdiag_stays_in_blocks():
    k = 8
    row, col, _, _ = support.sample_support(64, 48, 300, seed=3, mode=support.BLOCKDIAG, k=k)
    assert np.all(row // (64 // k) == col // (48 // k))


def test_zipf_row_frequencies():
    rows, s = 50, 1.1
    row, _, _, _ = support.sample_support(rows, 1_000_000, 20000, seed=5, mode=support.ZIPF_ROWS, zipf_s=s)
    p = np.arange(1, rows + 1, dtype=np.float64) ** -s
    p /= p.sum()
    counts = np.bincount(row, minlength=rows)
    expected = p * len(row)
    # with 10^6 columns per row duplicate draws are negligible: binomial tolerance per row
    sd = np.sqrt(expected * (1 - p))
    assert np.all(np.abs(counts - expected) < 5 * sd + 3)


def test_uniform_rows_are_flat():
    row, col, _, _ = support.sample_support(16, 4096, 16000, seed=6)
    counts = np.bincount(row, minlength=16)
    assert np.all(np.abs(counts - 1000) < 5 * np.sqrt(1000))
    ccounts = np.bincount(col // 256, minlength=16)
    assert np.all(np.abs(ccounts - 1000) < 5 * np.sqrt(1000))


def test_seed_changes_support():
    a = support.sample_support(128, 128, 64, seed=1)[0:2]
    b = support.sample_support(128, 128, 64, seed=2)[0:2]
    assert not (np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1]))
