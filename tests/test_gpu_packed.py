"""GPU parity of the packed units of the two-token tcgen05 kernel.

Where a side has at most 64 groups (d <= 2048), one 128-lane tile of the
kernel carries P tokens per slot (P = min(8, 128 // max(G_in, G_out)); 5 at
768 x 768), so a unit is 2P tokens.  These cases check the packed kernel
against the fp64 oracle (bf16 bar: per element |g - r| <= 2e-2 max(|r|,
rms r), Frobenius <= 5e-3) at token counts that end on every residue of a
unit, and against the unpacked kernel (FRAMEFB_PACK=0): the analysis,
coefficient SpMM and synthesis of one token do not depend on its lane, so Y
and dX are bit-equal; dC sums the same products in another order.
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2608_26430_gb300 import framefb as ffb
from paper_2608_26430_gb300 import workloads as wl
from paper_2608_26430_gb300.batch import AdapterBatch
from tests.oracle_side import Expect, assert_bf16, host64

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
ALL = ffb.OP_FORWARD | ffb.OP_BACKWARD_DX | ffb.OP_GRAD_COEFF
PACKED = "tc2p_tile_kernel<{}>"


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_26430_gb300.build import build
    build()
    ffb.lib()


def check(batch, ops, js=None):
    torch.cuda.synchronize()
    for j in (range(len(batch.bufs)) if js is None else js):
        b = batch.bufs[j]
        e = Expect(batch, j)
        X, dY = host64(b.X), host64(b.dY)
        if ops & ffb.OP_FORWARD:
            assert_bf16(host64(b.Y), e.y(X, np.zeros((X.shape[0], b.spec.m))), what=f"Y[{j}]")
        if ops & ffb.OP_BACKWARD_DX:
            assert_bf16(host64(b.dX), e.dx(dY, np.zeros((dY.shape[0], b.spec.n))), what=f"dX[{j}]")
        if ops & ffb.OP_GRAD_COEFF:
            assert_bf16(host64(b.dC), e.dc(X, dY), what=f"dC[{j}]")


def run(batch, ops):
    ws = batch.workspace(ops)
    batch.run(ops, ws)
    torch.cuda.synchronize()


@pytest.mark.parametrize("N", [1, 4, 5, 6, 9, 10, 11, 19, 37, 101])
def test_roberta_packed_every_tail(N):
    """768 x 768 (P = 5, units of 10 tokens): every residue of N mod 10."""
    b = AdapterBatch(wl.WORKLOADS["roberta_base_qv"], DEV, N=N, indices=[0, 1, 7], ops=ALL)
    assert ffb.framefb_kernel_names(b.mats, ALL, b.dtype_code) == [PACKED.format(ALL)]
    run(b, ALL)
    check(b, ALL)


@pytest.mark.parametrize("ops", [ffb.OP_FORWARD, ffb.OP_BACKWARD_DX, ffb.OP_GRAD_COEFF,
                                 ffb.OP_BACKWARD_DX | ffb.OP_GRAD_COEFF, ALL])
def test_roberta_packed_every_mode(ops):
    b = AdapterBatch(wl.WORKLOADS["roberta_base_qv"], DEV, N=23, indices=[0, 5], ops=ops)
    assert ffb.framefb_kernel_names(b.mats, ops, b.dtype_code) == [PACKED.format(ops)]
    run(b, ops)
    check(b, ops)


@pytest.mark.parametrize("N", [37, 4096])
def test_packed_matches_unpacked(N, monkeypatch):
    """Y and dX bit-equal to the unpacked kernel; dC within fp32 reordering."""
    w = wl.WORKLOADS["roberta_base_qv"]
    out = []
    for pack in ("1", "0"):
        monkeypatch.setenv("FRAMEFB_PACK", pack)
        b = AdapterBatch(w, DEV, N=N, indices=list(range(6)), ops=ALL)
        names = ffb.framefb_kernel_names(b.mats, ALL, b.dtype_code)
        assert names == ([PACKED.format(ALL)] if pack == "1" else [f"tc2_tile_kernel<{ALL}>"])
        run(b, ALL)
        out.append([(x.Y.clone(), x.dX.clone(), x.dC.clone()) for x in b.bufs])
    for (y1, x1, c1), (y0, x0, c0) in zip(*out):
        assert torch.equal(y1, y0) and torch.equal(x1, x0)
        torch.testing.assert_close(c1, c0, rtol=1e-5, atol=1e-5 * float(c0.abs().max()))


@pytest.mark.parametrize("N", [23, 37])
def test_vit_pairs_grouped_into_launches(N):
    """768 x 768 (P = 5) and 768 <-> 3072 (P = 1) matrices in one call: the
    call launches each pair count's matrices together (packed, then not)."""
    w = wl.WORKLOADS["vit_b16_merge"]
    b = AdapterBatch(w, DEV, N=N, ops=ALL)
    assert ffb.framefb_kernel_names(b.mats, ALL, b.dtype_code) == [PACKED.format(ALL), f"tc2_tile_kernel<{ALL}>"]
    run(b, ALL)
    check(b, ALL, js=[0, 3, 4, 5, 6, 10, 11, 70, 71])


def expected_tc2(plan, ops=ALL):
    """Packed units for plans of at most 8 entries per chunk (EZ, EG)."""
    h = np.frombuffer(plan.image()[:128].tobytes(), dtype=np.int32)
    return PACKED.format(ops) if max(h[8], h[9]) <= 8 else f"tc2_tile_kernel<{ops}>"


@pytest.mark.parametrize("nnz,N", [(1000, 37), (1000, 4096), (2000, 37), (4096, 37)])
def test_zipf_rows_packed_fixups(nnz, N):
    """Zipf(1.1) rows at 768 x 768: overflow slots and fix-ups per pair (the
    4096-entry plan holds 16 entries per chunk: unpacked units)."""
    w = dataclasses.replace(wl.WORKLOADS["roberta_zipf"], nnz=nnz)
    b = AdapterBatch(w, DEV, N=N, ops=ALL)
    want = expected_tc2(b.plans[(768, 768)])
    assert (want == PACKED.format(ALL)) == (nnz <= 2000)
    assert ffb.framefb_kernel_names(b.mats, ALL, b.dtype_code) == [want]
    run(b, ALL)
    check(b, ALL)


def test_eight_pairs_at_256():
    """256 x 256 in bf16 (8 groups a side): P at its cap of 8, units of 16."""
    w = dataclasses.replace(wl.WORKLOADS["single_256_fp32"], dtype="bf16", nnz=200)
    for N in (3, 16, 45):
        b = AdapterBatch(w, DEV, N=N, ops=ALL)
        assert ffb.framefb_kernel_names(b.mats, ALL, b.dtype_code) == [PACKED.format(ALL)]
        run(b, ALL)
        check(b, ALL)


def test_packed_accumulates():
    """Y and dX are read-modify-written: a second call adds the same delta."""
    b = AdapterBatch(wl.WORKLOADS["roberta_base_qv"], DEV, N=29, indices=[2], ops=ALL)
    run(b, ALL)
    y1, x1 = b.bufs[0].Y.float().clone(), b.bufs[0].dX.float().clone()
    run(b, ALL)
    y2, x2 = b.bufs[0].Y.float(), b.bufs[0].dX.float()
    # bf16 rounding of the doubled values: within one bf16 ulp of 2 x delta
    torch.testing.assert_close(y2, 2 * y1, rtol=2 ** -7, atol=1e-6)
    torch.testing.assert_close(x2, 2 * x1, rtol=2 ** -7, atol=1e-6)
