"""GPU parity of the mixed-tenant forward (serving without merge): tokens in
segments of different tenants, each using its own coefficient values on the
shared support, against the oracle's forward with each tenant's C.

The two-token kernels take the segment table in their launch parameters
(units stay inside segments; the coefficient values follow the unit's
tenant); FRAMEFB_SEG_KERNEL=0, other kernels and tables of more than 256
segments run every (matrix, segment) as a matrix of its own.  Both give the
same arithmetic per token, so their Y are bit-equal."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import adapter
from paper_2608_26430_gb300 import framefb as ffb
from paper_2608_26430_gb300 import workloads as wl
from paper_2608_26430_gb300.batch import AdapterBatch
from tests.oracle_side import Expect, assert_bf16, host64

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_26430_gb300.build import build
    build()
    ffb.lib()


def with_tenants(b, idx, T, seed0=900):
    """Copies of the batch's descriptors whose c_val is [T][nnz] per matrix."""
    w = b.w
    cvals = [wl.normal((T, w.nnz), seed0 + i, w.c_std, device=DEV) for i in idx]
    mats = []
    for mat, cv in zip(b.mats, cvals):
        m2 = ffb.framefb_mat.from_buffer_copy(mat)
        m2.c_val = cv.data_ptr()
        mats.append(m2)
    return mats, cvals


@pytest.mark.parametrize("seg_kernel", ["1", "0"])
@pytest.mark.parametrize("kernel", ["tc2", "tile"])
def test_mixed_tenant_forward(kernel, seg_kernel, monkeypatch):
    monkeypatch.setenv("FRAMEFB_KERNEL", kernel)
    monkeypatch.setenv("FRAMEFB_SEG_KERNEL", seg_kernel)
    w = wl.WORKLOADS["vit_b16_merge"]
    idx = [0, 4, 5]  # 768 x 768, 768 -> 3072, 3072 -> 768
    N, T = 100, 3
    seg_start = [0, 7, 27, 28, 28, 61, 100]  # odd boundaries, a one-token and an empty segment
    seg_tenant = [2, 0, 1, 1, 0, 2]
    b = AdapterBatch(w, DEV, N=N, indices=idx, ops=ffb.OP_FORWARD)
    mats, cvals = with_tenants(b, idx, T)
    ffb.framefb_forward_tenants(mats, b.dtype_code, seg_start, seg_tenant, T)
    torch.cuda.synchronize()
    for j, bb in enumerate(b.bufs):
        e = Expect(b, j)
        X, Y = host64(bb.X), host64(bb.Y)
        for i, tn in enumerate(seg_tenant):
            r0, r1 = seg_start[i], seg_start[i + 1]
            if r1 == r0:
                continue
            C = adapter.dense_C(bb.spec.m, bb.spec.n, e.row, e.col, host64(cvals[j][tn]))
            ref = adapter.forward(X[r0:r1], np.zeros((r1 - r0, bb.spec.m)), e.Pin, e.Pout, C, e.scale)
            assert_bf16(Y[r0:r1], ref, what=f"matrix {j} segment {i} (tenant {tn})")


def segments(N, nseg, T, seed):
    """nseg segments over N tokens with random boundaries (empty and one-token
    segments included) and random tenants."""
    g = np.random.default_rng(seed)
    cuts = np.sort(g.integers(0, N + 1, size=nseg - 1))
    start = [0] + [int(c) for c in cuts] + [N]
    return start, [int(t) for t in g.integers(0, T, size=nseg)]


@pytest.mark.parametrize("wname,idx,N,nseg", [
    ("vit_b16_merge", list(range(12)), 1000, 37),     # packed 768^2 and unpacked 768 <-> 3072 launches
    ("roberta_base_qv", list(range(6)), 3000, 256),   # the largest table the launch parameters hold
    ("roberta_base_qv", [0, 1], 600, 257),            # one more: per-segment launches
    ("llama2_7b_qkvo", [0, 1], 333, 9),               # unpacked two-token kernel only
])
def test_segment_kernel_matches_per_segment_launches(wname, idx, N, nseg, monkeypatch):
    """In-kernel segment table against one launch per (matrix, segment):
    Y bit-equal, and a sample of segments against the oracle."""
    w = wl.WORKLOADS[wname]
    T = 5
    seg_start, seg_tenant = segments(N, nseg, T, seed=nseg)
    ys = []
    for mode in ("1", "0"):
        monkeypatch.setenv("FRAMEFB_SEG_KERNEL", mode)
        b = AdapterBatch(w, DEV, N=N, indices=idx, ops=ffb.OP_FORWARD)
        mats, cvals = with_tenants(b, idx, T)
        ffb.framefb_forward_tenants(mats, b.dtype_code, seg_start, seg_tenant, T)
        torch.cuda.synchronize()
        ys.append([bb.Y.clone() for bb in b.bufs])
    for y1, y0 in zip(*ys):
        assert torch.equal(y1, y0)
    for j in (0, len(idx) - 1):
        bb = b.bufs[j]
        e = Expect(b, j)
        X = host64(bb.X)
        Y = host64(ys[0][j])
        for i in sorted({0, nseg // 2, nseg - 1}):
            r0, r1 = seg_start[i], seg_start[i + 1]
            if r1 == r0:
                continue
            C = adapter.dense_C(bb.spec.m, bb.spec.n, e.row, e.col, host64(cvals[j][seg_tenant[i]]))
            ref = adapter.forward(X[r0:r1], np.zeros((r1 - r0, bb.spec.m)), e.Pin, e.Pout, C, e.scale)
            assert_bf16(Y[r0:r1], ref, what=f"matrix {j} segment {i}")
