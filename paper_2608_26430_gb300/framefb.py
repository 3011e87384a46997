"""Thin ctypes binding of libframefb (include/framefb.h).

Argument marshalling only: every step of the adapter path runs in the CUDA
kernels of libframefb.so.  PyTorch provides device memory and the current
stream.  There is no fallback: if the library is missing or fails to load,
every call raises.
"""
from __future__ import annotations

import ctypes as ct
import os
from typing import Iterable, Sequence

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libframefb.so")

FRAMEFB_OK, FRAMEFB_EINVAL, FRAMEFB_EUNSUPPORTED, FRAMEFB_ENOMEM, FRAMEFB_ECUDA, FRAMEFB_EWORKSPACE = 0, -1, -2, -3, -4, -5
FRAMEFB_F32, FRAMEFB_BF16 = 0, 1
SUPPORT_UNIFORM, SUPPORT_ZIPF_ROWS, SUPPORT_BLOCKDIAG = 0, 1, 2
OP_FORWARD, OP_BACKWARD_DX, OP_GRAD_COEFF = 1, 2, 4
THREADS = 256

EXPORTED = [
    "framefb_status_string", "framefb_abi_version", "framefb_frame_build", "framefb_frame_free",
    "framefb_support_build", "framefb_plan_build", "framefb_plan_bytes", "framefb_plan_data", "framefb_plan_free",
    "framefb_plan_parts",
    "framefb_workspace_size", "framefb_run", "framefb_forward", "framefb_backward_dx", "framefb_grad_coeff",
    "framefb_backward", "framefb_fused_fwd_bwd", "framefb_merge", "framefb_run_static_ws",
    "framefb_wait_timeouts", "framefb_adamw", "framefb_linear_warmup_lr", "framefb_forward_tenants",
    "framefb_kernel_names", "framefb_frame_dense_bytes", "framefb_frame_dense_pack",
]
STATIC_WS_BYTES = 8 << 20
ABI_VERSION = 2  # FRAMEFB_ABI_VERSION of the structs below


class FramefbError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} ({status})")


class framefb_frame_params(ct.Structure):
    _fields_ = [("k", ct.c_int32), ("rho", ct.c_int32), ("parseval", ct.c_int32)]


class framefb_frame(ct.Structure):
    _fields_ = [("d", ct.c_int32), ("k", ct.c_int32), ("rho", ct.c_int32), ("ncols", ct.c_int32),
                ("nnz", ct.c_int64), ("A", ct.c_double), ("scale", ct.c_double),
                ("csc_colptr", ct.POINTER(ct.c_int64)), ("csc_rowidx", ct.POINTER(ct.c_int32)),
                ("csc_val", ct.POINTER(ct.c_double)),
                ("csr_rowptr", ct.POINTER(ct.c_int64)), ("csr_colidx", ct.POINTER(ct.c_int32)),
                ("csr_val", ct.POINTER(ct.c_double)),
                ("ngroups", ct.c_int32), ("grp_row0", ct.POINTER(ct.c_int32)), ("grp_nrows", ct.POINTER(ct.c_int32)),
                ("dft_groups", ct.c_int32)]


class framefb_dev_frame(ct.Structure):
    _fields_ = [("d", ct.c_int32), ("k", ct.c_int32), ("rho", ct.c_int32), ("ncols", ct.c_int32),
                ("dft_groups", ct.c_int32), ("pad_", ct.c_int32),
                ("colptr", ct.c_void_p), ("rowidx", ct.c_void_p), ("val", ct.c_void_p), ("dense", ct.c_void_p)]


class framefb_mat(ct.Structure):
    _fields_ = [("N", ct.c_int32), ("n", ct.c_int32), ("m", ct.c_int32), ("pad_", ct.c_int32),
                ("X", ct.c_void_p), ("dX", ct.c_void_p), ("ldx", ct.c_int64),
                ("dY", ct.c_void_p), ("Y", ct.c_void_p), ("ldy", ct.c_int64),
                ("fin", ct.POINTER(framefb_dev_frame)), ("fout", ct.POINTER(framefb_dev_frame)),
                ("plan", ct.c_void_p), ("plan_dev", ct.c_void_p),
                ("c_val", ct.c_void_p), ("dC", ct.c_void_p), ("scale", ct.c_float), ("pad2_", ct.c_int32)]


class framefb_adamw_params(ct.Structure):
    _fields_ = [("lr", ct.c_float), ("beta1", ct.c_float), ("beta2", ct.c_float), ("eps", ct.c_float),
                ("weight_decay", ct.c_float)]


_lib = None


def lib() -> ct.CDLL:
    """The loaded libframefb.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2608_26430_gb300.build.build()")
        L = ct.CDLL(LIB_PATH)
        i32, i64, vp, sz = ct.c_int32, ct.c_int64, ct.c_void_p, ct.c_size_t
        L.framefb_status_string.restype = ct.c_char_p
        L.framefb_status_string.argtypes = [i32]
        L.framefb_abi_version.restype = i32
        L.framefb_frame_build.restype = i32
        L.framefb_frame_build.argtypes = [i32, ct.POINTER(framefb_frame_params), ct.POINTER(framefb_frame)]
        L.framefb_frame_dense_bytes.restype = sz
        L.framefb_frame_dense_bytes.argtypes = [ct.POINTER(framefb_frame)]
        L.framefb_frame_dense_pack.restype = i32
        L.framefb_frame_dense_pack.argtypes = [ct.POINTER(framefb_frame), vp, sz]
        L.framefb_frame_free.restype = None
        L.framefb_frame_free.argtypes = [ct.POINTER(framefb_frame)]
        L.framefb_support_build.restype = i32
        L.framefb_support_build.argtypes = [i32, i32, i64, ct.c_uint64, i32, ct.c_double, i32, vp, vp, vp, vp]
        L.framefb_plan_build.restype = i32
        L.framefb_plan_build.argtypes = [ct.POINTER(framefb_frame), ct.POINTER(framefb_frame), vp, vp, i64,
                                         ct.POINTER(vp)]
        L.framefb_plan_bytes.restype = sz
        L.framefb_plan_bytes.argtypes = [vp]
        L.framefb_plan_parts.restype = i32
        L.framefb_plan_parts.argtypes = [vp, ct.POINTER(framefb_plan_part), i32]
        L.framefb_plan_data.restype = vp
        L.framefb_plan_data.argtypes = [vp]
        L.framefb_plan_free.restype = None
        L.framefb_plan_free.argtypes = [vp]
        L.framefb_workspace_size.restype = sz
        L.framefb_workspace_size.argtypes = [ct.POINTER(framefb_mat), i32, i32]
        L.framefb_run.restype = i32
        L.framefb_run.argtypes = [ct.POINTER(framefb_mat), i32, i32, i32, vp, sz, vp]
        for name in ("framefb_forward", "framefb_backward_dx", "framefb_grad_coeff", "framefb_backward",
                     "framefb_fused_fwd_bwd"):
            f = getattr(L, name)
            f.restype = i32
            f.argtypes = [ct.POINTER(framefb_mat), i32, i32, vp, sz, vp]
        L.framefb_kernel_names.restype = i32
        L.framefb_kernel_names.argtypes = [ct.POINTER(framefb_mat), i32, i32, i32, ct.c_char_p, sz]
        L.framefb_run_static_ws.restype = i32
        L.framefb_run_static_ws.argtypes = [ct.POINTER(framefb_mat), i32, i32, i32, vp]
        L.framefb_wait_timeouts.restype = i32
        L.framefb_wait_timeouts.argtypes = [ct.POINTER(ct.c_uint32)]
        L.framefb_merge.restype = i32
        L.framefb_merge.argtypes = [vp, i32, i32, i32, i64, ct.POINTER(framefb_dev_frame),
                                    ct.POINTER(framefb_dev_frame), vp, vp, vp, i32, ct.c_float, vp, vp]
        L.framefb_forward_tenants.restype = i32
        L.framefb_forward_tenants.argtypes = [ct.POINTER(framefb_mat), i32, i32, vp, vp, i32, i32, vp]
        L.framefb_adamw.restype = i32
        L.framefb_adamw.argtypes = [vp, vp, vp, vp, i64, ct.POINTER(framefb_adamw_params), i64, vp]
        L.framefb_linear_warmup_lr.restype = ct.c_double
        L.framefb_linear_warmup_lr.argtypes = [i64, i64, i64, ct.c_double]
        if L.framefb_abi_version() != ABI_VERSION:
            raise RuntimeError(f"{LIB_PATH} has ABI version {L.framefb_abi_version()}, the binding expects "
                               f"{ABI_VERSION}: rebuild it")
        _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().framefb_status_string(int(status)).decode()


def _check(status: int, what: str) -> None:
    if status != FRAMEFB_OK:
        raise FramefbError(status, what)


# ---------------------------------------------------------------------------
# S1 frames
# ---------------------------------------------------------------------------
class Frame:
    """Host frame built by framefb_frame_build (the C struct owns its arrays)."""

    def __init__(self, d: int, k: int, rho: int, parseval: bool = True):
        self._s = framefb_frame()
        p = framefb_frame_params(k, rho, 1 if parseval else 0)
        _check(lib().framefb_frame_build(d, ct.byref(p), ct.byref(self._s)), "framefb_frame_build")

    def __del__(self):
        if _lib is not None and getattr(self, "_s", None) is not None:
            _lib.framefb_frame_free(ct.byref(self._s))

    def __getattr__(self, name):
        if name in ("d", "k", "rho", "ncols", "nnz", "A", "scale", "ngroups", "dft_groups"):
            return getattr(self._s, name)
        raise AttributeError(name)

    @property
    def struct(self):
        return self._s

    def csc(self):
        s = self._s
        return (np.ctypeslib.as_array(s.csc_colptr, (s.ncols + 1,)).copy(),
                np.ctypeslib.as_array(s.csc_rowidx, (s.nnz,)).copy(),
                np.ctypeslib.as_array(s.csc_val, (s.nnz,)).copy())

    def csr(self):
        s = self._s
        return (np.ctypeslib.as_array(s.csr_rowptr, (s.d + 1,)).copy(),
                np.ctypeslib.as_array(s.csr_colidx, (s.nnz,)).copy(),
                np.ctypeslib.as_array(s.csr_val, (s.nnz,)).copy())

    def groups(self):
        s = self._s
        return (np.ctypeslib.as_array(s.grp_row0, (s.ngroups,)).copy(),
                np.ctypeslib.as_array(s.grp_nrows, (s.ngroups,)).copy())

    @property
    def structured(self) -> bool:
        """True when the structured kernels take this frame (k = 16, k*rho = d)."""
        s = self._s
        return bool(s.dft_groups) and s.k == 16 and s.ncols == s.d and s.d % 32 == 0

    def dense_image(self) -> np.ndarray:
        """The dense operand image of the frame (framefb_frame_dense_pack)."""
        n = int(lib().framefb_frame_dense_bytes(ct.byref(self._s)))
        out = np.zeros(max(n, 1), dtype=np.uint8)
        _check(lib().framefb_frame_dense_pack(ct.byref(self._s), out.ctypes.data, n), "framefb_frame_dense_pack")
        return out[:n]

    def to_device(self, device) -> "DevFrame":
        return DevFrame(self, device)


def framefb_frame_build(d: int, k: int, rho: int, parseval: bool = True) -> Frame:
    return Frame(d, k, rho, parseval)


class DevFrame:
    """fp32 device copy of a frame's CSC arrays plus the framefb_dev_frame view;
    frames outside the structured kernels also get their dense operand image
    (or always, with dense=True)."""

    def __init__(self, frame: Frame, device, dense: bool | None = None):
        import torch
        colptr, rowidx, val = frame.csc()
        self.colptr = torch.from_numpy(colptr).to(device)
        self.rowidx = torch.from_numpy(rowidx).to(device)
        self.val = torch.from_numpy(val.astype(np.float32)).to(device)
        self.dense = None
        if dense if dense is not None else not frame.structured:
            self.dense = torch.from_numpy(frame.dense_image()).to(device)
        self.struct = framefb_dev_frame(frame.d, frame.k, frame.rho, frame.ncols, frame.dft_groups, 0,
                                        self.colptr.data_ptr(), self.rowidx.data_ptr(), self.val.data_ptr(),
                                        _ptr(self.dense))


# ---------------------------------------------------------------------------
# S2 support and plan
# ---------------------------------------------------------------------------
def framefb_support_build(rows: int, cols: int, nnz: int, seed: int, mode: int = SUPPORT_UNIFORM,
                          zipf_s: float = 1.1, k: int = 1):
    row = np.zeros(max(nnz, 1), dtype=np.int32)
    col = np.zeros(max(nnz, 1), dtype=np.int32)
    rowptr = np.zeros(rows + 1, dtype=np.int64)
    perm = np.zeros(max(nnz, 1), dtype=np.int32)
    _check(lib().framefb_support_build(rows, cols, nnz, seed, mode, zipf_s, k, row.ctypes.data, col.ctypes.data,
                                       rowptr.ctypes.data, perm.ctypes.data), "framefb_support_build")
    return row[:nnz], col[:nnz], rowptr, perm[:nnz]


class framefb_plan_part(ct.Structure):
    _fields_ = [("image_offset", ct.c_int64), ("image_bytes", ct.c_int64), ("q_offset", ct.c_int64),
                ("nnz", ct.c_int32), ("n0", ct.c_int32), ("m0", ct.c_int32), ("n", ct.c_int32), ("m", ct.c_int32)]


class Plan:
    """Host plan handle (framefb_plan_build) and its device image bytes."""

    def __init__(self, fin: Frame, fout: Frame, row: np.ndarray, col: np.ndarray):
        row = np.ascontiguousarray(row, dtype=np.int32)
        col = np.ascontiguousarray(col, dtype=np.int32)
        self.nnz = int(row.size)
        h = ct.c_void_p()
        _check(lib().framefb_plan_build(ct.byref(fin.struct), ct.byref(fout.struct), row.ctypes.data,
                                        col.ctypes.data, self.nnz, ct.byref(h)), "framefb_plan_build")
        self.handle = h

    def __del__(self):
        if _lib is not None and getattr(self, "handle", None):
            _lib.framefb_plan_free(self.handle)
            self.handle = None

    def image(self) -> np.ndarray:
        n = lib().framefb_plan_bytes(self.handle)
        ptr = lib().framefb_plan_data(self.handle)
        return np.ctypeslib.as_array(ct.cast(ptr, ct.POINTER(ct.c_uint8)), (n,)).copy()

    def parts(self) -> list:
        """Descriptors of the plan's parts (framefb_plan_parts; [] when the
        fused kernels take the plan whole)."""
        n = lib().framefb_plan_parts(self.handle, None, 0)
        arr = (framefb_plan_part * max(n, 1))()
        lib().framefb_plan_parts(self.handle, arr, n)
        return [{f: getattr(arr[i], f) for f, _ in framefb_plan_part._fields_} for i in range(n)]

    def to_device(self, device):
        import torch
        return torch.from_numpy(self.image()).to(device)


def framefb_plan_build(fin: Frame, fout: Frame, row, col) -> Plan:
    return Plan(fin, fout, row, col)


# ---------------------------------------------------------------------------
# S3-S7 device entry points
# ---------------------------------------------------------------------------
def _ptr(t) -> int:
    return 0 if t is None else int(t.data_ptr())


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.bfloat16:
        return FRAMEFB_BF16
    if t.dtype == torch.float32:
        return FRAMEFB_F32
    raise TypeError(f"unsupported activation dtype {t.dtype}")


def make_mat(fin: DevFrame, fout: DevFrame, plan: Plan, plan_dev, c_val, scale: float, N: int,
             X=None, dX=None, dY=None, Y=None, dC=None, ldx: int | None = None, ldy: int | None = None) -> framefb_mat:
    """Descriptor of one adapted matrix over caller-owned torch tensors."""
    n, m = fin.struct.d, fout.struct.d
    if ldx is None:
        ldx = X.stride(0) if X is not None else (dX.stride(0) if dX is not None else n)
    if ldy is None:
        ldy = dY.stride(0) if dY is not None else (Y.stride(0) if Y is not None else m)
    return framefb_mat(N, n, m, 0, _ptr(X), _ptr(dX), ldx, _ptr(dY), _ptr(Y), ldy,
                       ct.pointer(fin.struct), ct.pointer(fout.struct), plan.handle.value, _ptr(plan_dev),
                       _ptr(c_val), _ptr(dC), float(scale), 0)


def _mats_array(mats: Sequence[framefb_mat]):
    arr = (framefb_mat * max(len(mats), 1))()
    for i, m in enumerate(mats):
        arr[i] = m
    return arr


def _stream(stream) -> int:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


def framefb_workspace_size(mats: Sequence[framefb_mat], ops: int) -> int:
    return int(lib().framefb_workspace_size(_mats_array(mats), len(mats), ops))


def workspace(mats: Sequence[framefb_mat], ops: int, device):
    """Caller-side workspace tensor (torch allocation) for a run."""
    import torch
    n = framefb_workspace_size(mats, ops)
    return torch.empty(max(n, 256), dtype=torch.uint8, device=device) if n > 0 else None


def framefb_run(mats: Sequence[framefb_mat], ops: int, dtype: int, ws=None, stream=None) -> None:
    arr = _mats_array(mats)
    wsp = _ptr(ws)
    wsb = 0 if ws is None else ws.numel() * ws.element_size()
    _check(lib().framefb_run(arr, len(mats), ops, dtype, wsp, wsb, _stream(stream)), "framefb_run")


def framefb_kernel_names(mats: Sequence[framefb_mat], ops: int, dtype: int) -> list:
    """Tile kernels framefb_run would launch for these matrices (no launch)."""
    buf = ct.create_string_buffer(1024)
    _check(lib().framefb_kernel_names(_mats_array(mats), len(mats), ops, dtype, buf, len(buf)),
           "framefb_kernel_names")
    v = buf.value.decode()
    return v.split(",") if v else []


def framefb_run_static_ws(mats: Sequence[framefb_mat], ops: int, dtype: int, stream=None) -> None:
    """framefb_run on the library's static device workspace (no allocation by anyone)."""
    arr = _mats_array(mats)
    _check(lib().framefb_run_static_ws(arr, len(mats), ops, dtype, _stream(stream)), "framefb_run_static_ws")


def framefb_forward(mats, dtype, ws=None, stream=None):
    framefb_run(mats, OP_FORWARD, dtype, ws, stream)


def framefb_forward_tenants(mats: Sequence[framefb_mat], dtype: int, seg_start, seg_tenant, ntenants: int,
                            stream=None) -> None:
    """Mixed-tenant forward: tokens [seg_start[i], seg_start[i+1]) use tenant
    seg_tenant[i]'s coefficient values (each mat's c_val is [ntenants][nnz])."""
    nseg = len(seg_tenant)
    if len(seg_start) != nseg + 1:
        raise ValueError("seg_start needs one more entry than seg_tenant")
    starts = (ct.c_int32 * (nseg + 1))(*[int(x) for x in seg_start])
    tenants = (ct.c_int32 * max(nseg, 1))(*[int(x) for x in seg_tenant])
    arr = _mats_array(mats)
    _check(lib().framefb_forward_tenants(arr, len(mats), dtype, starts, tenants, nseg, int(ntenants),
                                         _stream(stream)), "framefb_forward_tenants")


def framefb_backward_dx(mats, dtype, ws=None, stream=None):
    framefb_run(mats, OP_BACKWARD_DX, dtype, ws, stream)


def framefb_grad_coeff(mats, dtype, ws=None, stream=None):
    framefb_run(mats, OP_GRAD_COEFF, dtype, ws, stream)


def framefb_backward(mats, dtype, ws=None, stream=None):
    framefb_run(mats, OP_BACKWARD_DX | OP_GRAD_COEFF, dtype, ws, stream)


def framefb_fused_fwd_bwd(mats, dtype, ws=None, stream=None):
    framefb_run(mats, OP_FORWARD | OP_BACKWARD_DX | OP_GRAD_COEFF, dtype, ws, stream)


def framefb_merge(W0, fin: DevFrame, fout: DevFrame, plan: Plan, plan_dev, c_vals, T: int, scale: float, Wout,
                  stream=None) -> None:
    m, n = W0.shape
    _check(lib().framefb_merge(_ptr(W0), _dtype_code(W0), m, n, W0.stride(0), ct.byref(fin.struct),
                               ct.byref(fout.struct), plan.handle.value, _ptr(plan_dev), _ptr(c_vals), T,
                               float(scale), _ptr(Wout), _stream(stream)), "framefb_merge")


def framefb_adamw(param, grad, m, v, step: int, lr: float, beta1: float = 0.9, beta2: float = 0.999,
                  eps: float = 1e-8, weight_decay: float = 0.01, n: int | None = None, stream=None) -> None:
    """One AdamW step on fp32 device tensors (param, m, v updated in place)."""
    if n is None:
        n = param.numel()
    hp = framefb_adamw_params(float(lr), float(beta1), float(beta2), float(eps), float(weight_decay))
    _check(lib().framefb_adamw(_ptr(param), _ptr(grad), _ptr(m), _ptr(v), int(n), ct.byref(hp), int(step),
                               _stream(stream)), "framefb_adamw")


def framefb_linear_warmup_lr(i: int, total: int, warmup: int, lr_max: float) -> float:
    return float(lib().framefb_linear_warmup_lr(int(i), int(total), int(warmup), float(lr_max)))


def framefb_wait_timeouts() -> int:
    n = ct.c_uint32(0)
    _check(lib().framefb_wait_timeouts(ct.byref(n)), "framefb_wait_timeouts")
    return int(n.value)


def exported_symbols(names: Iterable[str] = EXPORTED) -> dict:
    """Which of the header's entry points the loaded library exports."""
    L = lib()
    return {n: hasattr(L, n) for n in names}
