"""Assemble the library's inputs for a batch of adapted matrices.

Frames (one per distinct dimension, shared across layers -- Sec. 3.4), the
support and its plan (one per distinct (m, n) shape, shared across layers --
Sec. 3.3), device copies of both, per-matrix C values and activation buffers,
and the framefb_mat descriptors.  Every computation of the method happens in
libframefb; this module only allocates (torch) and marshals.
"""
from __future__ import annotations

from dataclasses import dataclass

from . import framefb as ffb
from . import workloads as wl


@dataclass
class MatBuffers:
    spec: wl.MatSpec
    scale: float
    c_val: object
    X: object = None
    dY: object = None
    Y: object = None
    dX: object = None
    dC: object = None


class AdapterBatch:
    """All inputs of one workload on one device.

    N: tokens per matrix (defaults to the workload's); indices: which of the
    workload's matrices to include (defaults to all); alias_inputs: share X by
    input dimension and dY by output dimension (read-only inputs of a model
    whose layers see the same shapes); y_init / dx_init: "zeros" or "random".
    The coefficient values of all matrices are rows of one [matrices x nnz]
    tensor ``C`` (and their gradients rows of ``dC``), so that one optimiser
    call covers them all.
    """

    def __init__(self, w: wl.Workload, device, N: int | None = None, indices=None, alias_inputs: bool = False,
                 y_init: str = "zeros", unit_scale: bool = False, ops: int = 7):
        import torch
        self.w = w
        self.device = device
        self.N = w.N if N is None else N
        self.indices = list(range(len(w.mats))) if indices is None else list(indices)
        self.dtype = wl.torch_dtype(w)
        self.dtype_code = ffb.FRAMEFB_F32 if w.dtype == "f32" else ffb.FRAMEFB_BF16
        self.frames = {d: ffb.Frame(d, *wl.frame_params(w, d), parseval=True) for d in w.dims()}
        self.dev_frames = {d: f.to_device(device) for d, f in self.frames.items()}
        # one support and plan per shape (shared across layers, Sec. 3.3), or
        # per matrix for per-layer supports
        self.supports, self.plans, self.plan_dev = {}, {}, {}
        self.keys = [wl.support_key(w, i) for i in self.indices]
        for key, i in zip(self.keys, self.indices):
            if key in self.plans:
                continue
            m, n = key[0], key[1]
            km, kn = self.frames[m].ncols, self.frames[n].ncols  # C is K_m x K_n
            row, col, _, _ = ffb.framefb_support_build(km, kn, w.nnz, wl.support_seed_of(w, i), w.support_mode,
                                                       w.zipf_s, w.k)
            self.supports[key] = (row, col)
            self.plans[key] = ffb.Plan(self.frames[n], self.frames[m], row, col)
            self.plan_dev[key] = self.plans[key].to_device(device)
        shared_x, shared_dy = {}, {}
        self.C = torch.stack([wl.c_values(w, i, device) for i in self.indices]) if self.indices else None
        self.dC = (torch.full((len(self.indices), w.nnz), float("nan"), dtype=torch.float32, device=device)
                   if ops & ffb.OP_GRAD_COEFF and self.indices else None)
        self.bufs = []
        for r, i in enumerate(self.indices):
            spec = w.mats[i]
            s = 1.0 if unit_scale else wl.scale_of(w, spec)
            b = MatBuffers(spec, s, self.C[r])
            if ops & (ffb.OP_FORWARD | ffb.OP_GRAD_COEFF):
                if alias_inputs:
                    if spec.n not in shared_x:
                        shared_x[spec.n] = self._pad(wl.x_input(w, i, self.N, device))
                    b.X = shared_x[spec.n]
                else:
                    b.X = self._pad(wl.x_input(w, i, self.N, device))
            if ops & (ffb.OP_BACKWARD_DX | ffb.OP_GRAD_COEFF):
                if alias_inputs:
                    if spec.m not in shared_dy:
                        shared_dy[spec.m] = self._pad(wl.dy_input(w, i, self.N, device))
                    b.dY = shared_dy[spec.m]
                else:
                    b.dY = self._pad(wl.dy_input(w, i, self.N, device))
            if ops & ffb.OP_FORWARD:
                b.Y = self._pad(self._init((self.N, spec.m), y_init, i, 7))
            if ops & ffb.OP_BACKWARD_DX:
                b.dX = self._pad(self._init((self.N, spec.n), y_init, i, 8))
            if ops & ffb.OP_GRAD_COEFF:
                b.dC = self.dC[r]
            self.bufs.append(b)
        self.mats = [self._mat(b, key) for b, key in zip(self.bufs, self.keys)]

    def _pad(self, t):
        """t itself, or a view of it inside rows padded to 16 bytes (the
        interface's row alignment) when its width needs it."""
        import torch
        d = t.shape[1]
        per = 16 // t.element_size()
        ld = (d + per - 1) // per * per
        if ld == d:
            return t
        p = torch.zeros((t.shape[0], ld), dtype=t.dtype, device=t.device)
        p[:, :d] = t
        return p[:, :d]

    def _init(self, shape, kind, i, salt):
        import torch
        if kind == "zeros":
            return torch.zeros(shape, dtype=self.dtype, device=self.device)
        return wl.normal(shape, 10000 * salt + i, 1.0, self.dtype, self.device)

    def _mat(self, b: MatBuffers, key):
        spec = b.spec
        def ld(*ts):
            for t in ts:
                if t is not None:
                    return t.stride(0)
            return None
        return ffb.make_mat(self.dev_frames[spec.n], self.dev_frames[spec.m], self.plans[key], self.plan_dev[key],
                            b.c_val, b.scale, self.N, X=b.X, dX=b.dX, dY=b.dY, Y=b.Y, dC=b.dC,
                            ldx=ld(b.X, b.dX) or spec.n, ldy=ld(b.dY, b.Y) or spec.m)

    def workspace(self, ops: int):
        return ffb.workspace(self.mats, ops, self.device)

    def run(self, ops: int, ws=None, stream=None):
        ffb.framefb_run(self.mats, ops, self.dtype_code, ws, stream)
