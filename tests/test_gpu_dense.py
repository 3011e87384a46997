"""GPU parity of the dense path (frames outside the structured kernels)
through the C ABI, against the fp64 oracle.

The paper's own regime rho = 2 (Phi a dense realified DFT of size d/2) at
RoBERTa and LLaMA-2 shapes, and redundant tight fusion frames with T blocks
(k*rho > d) at small odd shapes, with the bf16 bar: per element
|g - r| <= 2e-2 max(|r|, rms r), Frobenius-relative <= 5e-3.
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


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_26430_gb300.build import build
    build()
    ffb.lib()


def check(batch, ops, js=None, rows=None, Y0=None, dX0=None):
    torch.cuda.synchronize()
    for j in (range(len(batch.bufs)) if js is None else js):
        b, e = batch.bufs[j], Expect(batch, j)
        X, dY = host64(b.X), host64(b.dY)
        sel = np.arange(batch.N) if rows is None else rows
        tsel = torch.from_numpy(sel).to(DEV)
        if ops & ffb.OP_FORWARD:
            y0 = np.zeros((sel.size, b.spec.m)) if Y0 is None else Y0[j][sel]
            assert_bf16(host64(b.Y[tsel]), e.y(X[sel], y0), what=f"Y[{j}]")
        if ops & ffb.OP_BACKWARD_DX:
            x0 = np.zeros((sel.size, b.spec.n)) if dX0 is None else dX0[j][sel]
            assert_bf16(host64(b.dX[tsel]), e.dx(dY[sel], x0), what=f"dX[{j}]")
        if ops & ffb.OP_GRAD_COEFF:
            assert_bf16(host64(b.dC), e.dc(X, dY), what=f"dC[{j}]")


def run(batch, ops):
    ws = batch.workspace(ops)
    batch.run(ops, ws)
    torch.cuda.synchronize()


@pytest.mark.parametrize("ops", [ffb.OP_FORWARD, ffb.OP_BACKWARD_DX, ffb.OP_GRAD_COEFF,
                                 ffb.OP_BACKWARD_DX | ffb.OP_GRAD_COEFF, ALL])
@pytest.mark.parametrize("N", [1, 37, 300])
def test_rho2_roberta_shapes(N, ops):
    """rho = 2 at d = 768: one dense DFT_384 per token (K = 768 columns); the
    token counts cover one partial tile, a ragged pair and several tiles."""
    w = wl.WORKLOADS["roberta_rho2"]
    b = AdapterBatch(w, DEV, N=N, indices=[0, 1], ops=ops)
    names = ffb.framefb_kernel_names(b.mats, ops, b.dtype_code)
    assert names[0] == "dense_gemm_kernel<bf16_hilo>"
    run(b, ops)
    check(b, ops)


def test_rho2_llama_shape():
    """rho = 2 at d = 4096 (dense DFT_2048 per token), two token tiles."""
    w = wl.WORKLOADS["llama2_rho2"]
    b = AdapterBatch(w, DEV, N=200, indices=[0], ops=ALL)
    run(b, ALL)
    check(b, ALL)


@pytest.mark.parametrize("ops", [ffb.OP_FORWARD, ffb.OP_BACKWARD_DX, ffb.OP_GRAD_COEFF, ALL])
def test_tblock_frames_nonsquare(ops):
    """Redundant frames with T blocks (k*rho > d): (40, 7, 8) -> (22, 6, 6),
    (46, 10, 10) square and (22, 6, 6) -> (40, 7, 8); feature counts that are
    not multiples of 8 sit in rows padded to 16 bytes."""
    w = wl.WORKLOADS["tblock_tff"]
    b = AdapterBatch(w, DEV, ops=ops)
    run(b, ops)
    check(b, ops)


def test_dense_accumulates_and_entry_points_agree():
    w = wl.WORKLOADS["roberta_rho2"]
    fused = AdapterBatch(w, DEV, N=150, indices=[0, 1], ops=ALL, y_init="random")
    Y0 = [host64(x.Y) for x in fused.bufs]
    dX0 = [host64(x.dX) for x in fused.bufs]
    run(fused, ALL)
    check(fused, ALL, Y0=Y0, dX0=dX0)
    sep = AdapterBatch(w, DEV, N=150, indices=[0, 1], ops=ALL, y_init="random")
    ws = sep.workspace(ALL)
    ffb.framefb_forward(sep.mats, sep.dtype_code, ws)
    ffb.framefb_backward_dx(sep.mats, sep.dtype_code, ws)
    ffb.framefb_grad_coeff(sep.mats, sep.dtype_code, ws)
    torch.cuda.synchronize()
    for a, c in zip(fused.bufs, sep.bufs):
        assert torch.equal(a.Y, c.Y) and torch.equal(a.dX, c.dX) and torch.equal(a.dC, c.dC)


def test_structured_and_dense_matrices_in_one_call():
    """One framefb_run over matrices of both paths (DFT_16-group frames and
    rho = 2 frames): each path gets its matrices, the workspace is shared."""
    ws_ = wl.WORKLOADS["roberta_base_qv"]
    wd = wl.WORKLOADS["roberta_rho2"]
    bs = AdapterBatch(ws_, DEV, N=64, indices=[0, 1], ops=ALL)
    bd = AdapterBatch(wd, DEV, N=64, indices=[0, 1], ops=ALL)
    mats = [bs.mats[0], bd.mats[0], bs.mats[1], bd.mats[1]]
    names = ffb.framefb_kernel_names(mats, ALL, ffb.FRAMEFB_BF16)
    assert "tc2p_tile_kernel<7>" in names and "dense_gemm_kernel<tf32>" in names
    ws = ffb.workspace(mats, ALL, DEV)
    ffb.framefb_run(mats, ALL, ffb.FRAMEFB_BF16, ws)
    check(bs, ALL)
    check(bd, ALL)


def test_token_chunks_of_the_workspace():
    """More tokens than one workspace pass holds (8192): two chunks, dC summed
    over both in a fixed order."""
    w = dataclasses.replace(wl.WORKLOADS["roberta_rho2"], N=8192 + 77)
    b = AdapterBatch(w, DEV, indices=[0], ops=ALL)
    run(b, ALL)
    rows = np.unique(np.concatenate([[0, 8191, 8192, w.N - 1], np.random.default_rng(2).choice(w.N, 60, replace=False)]))
    check(b, ALL, rows=rows)


def test_dense_path_refusals():
    w = wl.WORKLOADS["tblock_tff"]
    b = AdapterBatch(w, DEV, N=8, indices=[0], ops=ALL)
    with pytest.raises(ffb.FramefbError) as e:        # the dense path takes bf16 activations
        ffb.framefb_run(b.mats, ALL, ffb.FRAMEFB_F32, b.workspace(ALL))
    assert e.value.status == ffb.FRAMEFB_EUNSUPPORTED
    with pytest.raises(ffb.FramefbError) as e:        # no workspace
        ffb.framefb_run(b.mats, ALL, ffb.FRAMEFB_BF16, None)
    assert e.value.status == ffb.FRAMEFB_EWORKSPACE
    bad = ffb.framefb_mat.from_buffer_copy(b.mats[0])
    bad.n = 48                                          # features differ from the plan's frame
    with pytest.raises(ffb.FramefbError) as e:
        ffb.framefb_run([bad], ALL, ffb.FRAMEFB_BF16, b.workspace(ALL))
    assert e.value.status == ffb.FRAMEFB_EINVAL
