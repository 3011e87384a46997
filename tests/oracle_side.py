"""Oracle-side expectations for a batch built by paper_2608_26430_gb300.batch.

Only the oracle computes here: the support is re-drawn by oracle.support
from the workload's seed (the library's support is asserted equal), the
frames are the oracle's dense fp64 matrices, and the activations / C values
are the seeded inputs both sides share (bf16 inputs are exact in fp64).
"""
from functools import lru_cache

import numpy as np

from oracle import adapter, frames, support
from paper_2608_26430_gb300 import workloads as wl


@lru_cache(maxsize=8)
def frame(d: int, k: int, rho: int | None = None) -> np.ndarray:
    return frames.real_frame(d, k, d // k if rho is None else rho, parseval=True)


@lru_cache(maxsize=16)
def oracle_support(m, n, nnz, seed, mode, zipf_s, k):
    return support.sample_support(m, n, nnz, seed, mode, zipf_s, k)


def host64(t):
    return None if t is None else t.detach().float().cpu().double().numpy()


class Expect:
    """Dense oracle quantities of matrix j of `batch`."""

    def __init__(self, batch, j):
        w, b = batch.w, batch.bufs[j]
        spec = b.spec
        self.spec, self.scale = spec, b.scale
        seed = wl.support_seed_of(w, batch.indices[j])
        km, kn = wl.coef_dims(w, spec)
        row, col, _, _ = oracle_support(km, kn, w.nnz, seed, w.support_mode, w.zipf_s, w.k)
        lrow, lcol = batch.supports[batch.keys[j]]
        assert np.array_equal(row, lrow) and np.array_equal(col, lcol), "support differs from the oracle's"
        self.row, self.col = row, col
        self.Pin = frame(spec.n, *wl.frame_params(w, spec.n))
        self.Pout = frame(spec.m, *wl.frame_params(w, spec.m))
        self.c = host64(b.c_val)
        self.C = adapter.dense_C(km, kn, row, col, self.c)
        self._dW = None

    @property
    def dW(self):
        if self._dW is None:
            self._dW = adapter.delta_w(self.Pout, self.C, self.Pin, self.scale)
        return self._dW

    def y(self, X, Y0):
        return adapter.forward(X, Y0, self.Pin, self.Pout, self.C, self.scale)

    def dx(self, dY, dX0):
        return adapter.backward_dx(dY, dX0, self.Pin, self.Pout, self.C, self.scale)

    def dc(self, X, dY):
        return adapter.grad_coeff(X, dY, self.Pin, self.Pout, self.scale, self.row, self.col)


def assert_f32(g, r, tol=1e-5, what=""):
    g, r = np.asarray(g, np.float64), np.asarray(r, np.float64)
    scale = np.max(np.abs(r)) if r.size else 0.0
    err = np.max(np.abs(g - r)) if r.size else 0.0
    assert err <= tol * max(scale, 1e-30), f"{what}: max err {err:.3e} vs max |ref| {scale:.3e}"


def assert_bf16(g, r, elem=2e-2, frob=5e-3, what=""):
    g, r = np.asarray(g, np.float64), np.asarray(r, np.float64)
    if r.size == 0:
        return
    rms = np.sqrt(np.mean(r * r))
    bound = elem * np.maximum(np.abs(r), rms)
    bad = np.abs(g - r) > bound
    assert not bad.any(), f"{what}: {bad.sum()} elements over the per-element bound, worst {np.max(np.abs(g - r) / np.maximum(bound, 1e-30)):.3f}x"
    rel = np.linalg.norm(g - r) / max(np.linalg.norm(r), 1e-30)
    assert rel <= frob, f"{what}: Frobenius-relative error {rel:.3e}"
