"""Pins of the oracle's frame construction against the paper and mathematics.

* the printed (6,3,11) worked example (Spectral Tetris F and the modulated TFF)
* UNTF properties of F and tightness P P^T = A I of the real frame
* the closed form for k*rho = d: analysis = inverse DFT_k (numpy.fft, "ortho"),
  synthesis = forward DFT_k, per group of 2k coordinates
"""
import math

import numpy as np
import pytest

from oracle import frames
from tests.goldens import load_omega_matrix, load_real_matrix


def test_spectral_tetris_matches_worked_example():
    F = frames.spectral_tetris(3, 11)
    want = load_real_matrix("st_F_3_11.txt")
    np.testing.assert_allclose(F, want, rtol=0, atol=1e-15)


def test_modulation_matches_worked_example_table():
    F = frames.spectral_tetris(3, 11)
    M = frames.modulated_frame(6, F)           # [k_i, r, j]
    got = np.concatenate([M[:, r, :] for r in range(3)], axis=0)  # row 6r + k_i
    want = load_omega_matrix("tff_6_3_11.txt", 6)
    assert got.shape == want.shape == (18, 11)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-14)


@pytest.mark.parametrize("rho_c,d_c", [(3, 11), (2, 5), (4, 9), (5, 23), (8, 64), (7, 30), (1, 2), (128, 2048)])
def test_untf_properties(rho_c, d_c):
    F = frames.spectral_tetris(rho_c, d_c)
    np.testing.assert_allclose(np.linalg.norm(F, axis=0), 1.0, atol=1e-14)
    np.testing.assert_allclose(F @ F.T, (d_c / rho_c) * np.eye(rho_c), atol=1e-12)


def test_spectral_tetris_rejects_too_few_columns():
    with pytest.raises(ValueError):
        frames.spectral_tetris(4, 7)


def test_modulation_rejects_too_few_subspaces():
    # widest row support of F(3,11) is 6 columns: k = 5 cannot separate them
    with pytest.raises(ValueError):
        frames.real_frame(22, 5, 6, parseval=False)


@pytest.mark.parametrize("d,k,rho", [(22, 6, 6), (256, 16, 16), (64, 8, 8), (768, 16, 48),
                                     (24, 4, 6), (46, 10, 10), (12, 2, 6), (40, 7, 8)])
def test_real_frame_is_tight(d, k, rho):
    P = frames.real_frame(d, k, rho, parseval=False)
    A = frames.frame_bound(d, k, rho)
    assert P.shape == (d, k * rho)
    np.testing.assert_allclose(np.linalg.norm(P, axis=0), 1.0, atol=1e-13)
    np.testing.assert_allclose(P @ P.T, A * np.eye(d), atol=1e-12)
    Pp = frames.real_frame(d, k, rho, parseval=True)
    np.testing.assert_allclose(Pp @ Pp.T, np.eye(d), atol=1e-12)
    # every subspace block P_i has orthonormal columns (P_i P_i^T is an orthogonal projection)
    for i in range(k):
        Pi = P[:, i * rho:(i + 1) * rho]
        np.testing.assert_allclose(Pi.T @ Pi, np.eye(rho), atol=1e-13)


def test_worked_example_real_bound():
    P = frames.real_frame(22, 6, 6, parseval=False)
    np.testing.assert_allclose(P @ P.T, (18.0 / 11.0) * np.eye(22), atol=1e-13)


# rho = d / k; the last three are the paper's own regime rho = 2 (one dense DFT_{d/2})
@pytest.mark.parametrize("d,k", [(256, 16), (64, 8), (96, 16), (48, 4), (40, 2), (64, 32), (256, 128), (12, 6)])
def test_closed_form_analysis_is_inverse_dft(d, k):
    rho = d // k
    P = frames.real_frame(d, k, rho, parseval=True)
    rng = np.random.default_rng(7)
    X = rng.standard_normal((5, d))
    V = X @ P
    rho_c = rho // 2
    for r in range(rho_c):
        z = X[:, 2 * r * k:2 * (r + 1) * k:2] + 1j * X[:, 2 * r * k + 1:2 * (r + 1) * k:2]
        f = np.fft.ifft(z, axis=1, norm="ortho")
        for i in range(k):
            np.testing.assert_allclose(V[:, i * rho + 2 * r], f[:, i].real, atol=1e-13)
            np.testing.assert_allclose(V[:, i * rho + 2 * r + 1], f[:, i].imag, atol=1e-13)


@pytest.mark.parametrize("d,k", [(256, 16), (64, 8), (64, 32)])
def test_closed_form_synthesis_is_forward_dft(d, k):
    rho = d // k
    P = frames.real_frame(d, k, rho, parseval=True)
    rng = np.random.default_rng(8)
    Z = rng.standard_normal((3, k * rho))
    Y = Z @ P.T
    for r in range(rho // 2):
        zeta = np.stack([Z[:, i * rho + 2 * r] + 1j * Z[:, i * rho + 2 * r + 1] for i in range(k)], axis=1)
        f = np.fft.fft(zeta, axis=1, norm="ortho")
        np.testing.assert_allclose(Y[:, 2 * r * k:2 * (r + 1) * k:2], f.real, atol=1e-13)
        np.testing.assert_allclose(Y[:, 2 * r * k + 1:2 * (r + 1) * k:2], f.imag, atol=1e-13)


@pytest.mark.parametrize("d,k,rho", [(256, 16, 16), (22, 6, 6), (40, 7, 8)])
def test_storage_pattern_covers_values(d, k, rho):
    P = frames.real_frame(d, k, rho)
    pat = frames.structural_pattern(d, k, rho)
    assert not np.any(P[~pat])                   # nothing outside the stored pattern
    colptr, rowidx, cval = frames.csc_from_dense(P, pat)
    rowptr, colidx, rval = frames.csr_from_dense(P, pat)
    assert colptr[-1] == rowptr[-1] == pat.sum()
    # CSC and CSR hold the same (row, col, value) triples
    csc = sorted(zip(rowidx.tolist(), np.repeat(np.arange(k * rho), np.diff(colptr)).tolist(), cval.tolist()))
    csr = sorted(zip(np.repeat(np.arange(d), np.diff(rowptr)).tolist(), colidx.tolist(), rval.tolist()))
    assert csc == csr


def test_dft_frame_groups_are_disjoint_blocks():
    d, k, rho = 256, 16, 16
    row0, nrows = frames.group_table(d, k, rho)
    assert list(row0) == [2 * k * r for r in range(rho // 2)]
    assert set(nrows.tolist()) == {2 * k}
    pat = frames.structural_pattern(d, k, rho)
    assert pat.sum() == d * 2 * k                 # structural zeros are stored
    P = frames.real_frame(d, k, rho)
    assert np.count_nonzero(P) < pat.sum()        # some stored values are exact zeros


def test_group_table_matches_printed_worked_example():
    # the printed F of the (6,3,11) walk-through has row supports columns 0-4,
    # 3-8 and 7-10 (T blocks straddle rows); a group covers the real
    # coordinates 2j, 2j+1 of its row's complex columns j
    F = load_real_matrix("st_F_3_11.txt")
    printed = [(int(np.nonzero(F[r])[0][0]), int(np.nonzero(F[r])[0][-1])) for r in range(3)]
    assert printed == [(0, 4), (3, 8), (7, 10)]
    row0, nrows = frames.group_table(22, 6, 6)
    assert row0.tolist() == [0, 6, 14]
    assert nrows.tolist() == [10, 12, 8]


@pytest.mark.parametrize("d,k,rho", [(22, 6, 6), (40, 7, 8), (46, 10, 10), (24, 4, 6), (256, 16, 16)])
def test_group_table_is_the_row_span_of_each_groups_columns(d, k, rho):
    # the columns {i*rho + 2r + s} of group r live exactly on the coordinates
    # [row0[r], row0[r] + nrows[r]): nothing outside, and both boundary
    # coordinate pairs used -- checked on the dense frame, so that an
    # off-by-one in the range (e.g. a T block's spill row) fails
    row0, nrows = frames.group_table(d, k, rho)
    P = frames.real_frame(d, k, rho, parseval=False)
    assert row0.size == nrows.size == rho // 2
    for r in range(rho // 2):
        cols = [i * rho + 2 * r + s for i in range(k) for s in (0, 1)]
        used = np.nonzero(np.any(P[:, cols] != 0, axis=1))[0]
        lo, hi = int(row0[r]), int(row0[r] + nrows[r])
        assert used.min() >= lo and used.max() < hi
        assert {used.min() // 2, used.max() // 2} == {lo // 2, hi // 2 - 1}
    # T-block frames: consecutive groups overlap by exactly the shared complex column pair
    sup = frames.row_supports(frames.spectral_tetris(rho // 2, d // 2))
    for r in range(rho // 2 - 1):
        overlap = max(0, sup[r][1] - sup[r + 1][0] + 1)
        assert overlap in (0, 2)
        assert (row0[r] + nrows[r] - row0[r + 1]) == 2 * overlap
