"""GPU parity of the mixed-tenant forward (serving without merge): tokens in
segments of different tenants, each using its own coefficient values on the
shared support, against the oracle's forward with each tenant's C."""
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


@pytest.mark.parametrize("kernel", ["tc2", "tile"])
def test_mixed_tenant_forward(kernel, monkeypatch):
    monkeypatch.setenv("FRAMEFB_KERNEL", kernel)
    w = wl.WORKLOADS["vit_b16_merge"]
    idx = [0, 4, 5]  # 768 x 768, 768 -> 3072, 3072 -> 768
    N, T = 100, 3
    seg_start = [0, 7, 27, 28, 28, 61, 100]  # odd boundaries, a one-token and an empty segment
    seg_tenant = [2, 0, 1, 1, 0, 2]
    b = AdapterBatch(w, DEV, N=N, indices=idx, ops=ffb.OP_FORWARD)
    cvals = [wl.normal((T, w.nnz), 900 + i, w.c_std, device=DEV) for i in idx]
    mats = []
    for mat, cv in zip(b.mats, cvals):
        m2 = ffb.framefb_mat.from_buffer_copy(mat)
        m2.c_val = cv.data_ptr()
        mats.append(m2)
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
