"""GPU parity of the CUDA path (through the C ABI) against the fp64 oracle.

Tolerances (stated for the adapter path): fp32 activations -- max |g - r| /
max |r| <= 1e-5; bf16 activations with fp32 accumulation -- per element
|g - r| <= 2e-2 max(|r|, rms(r)) and ||g - r||_F / ||r||_F <= 5e-3.
Deltas are checked with Y_in = dX_in = 0; accumulation is checked in fp32.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2608_26430_gb300 import framefb as ffb
from paper_2608_26430_gb300 import workloads as wl
from paper_2608_26430_gb300.batch import AdapterBatch
from tests.oracle_side import Expect, assert_bf16, assert_f32, host64

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


def check_batch(batch, ops, js=None, unit=None, rows=None):
    w = batch.w
    close = assert_f32 if w.dtype == "f32" else assert_bf16
    torch.cuda.synchronize()
    for j in (range(len(batch.bufs)) if js is None else js):
        b = batch.bufs[j]
        e = Expect(batch, j)
        X, dY = host64(b.X), host64(b.dY)
        sel = slice(None) if rows is None else rows
        if ops & ffb.OP_FORWARD:
            r = e.y(X[sel], np.zeros((X[sel].shape[0], b.spec.m)))
            close(host64(b.Y)[sel], r, what=f"Y[{j}]")
        if ops & ffb.OP_BACKWARD_DX:
            r = e.dx(dY[sel], np.zeros((dY[sel].shape[0], b.spec.n)))
            close(host64(b.dX)[sel], r, what=f"dX[{j}]")
        if ops & ffb.OP_GRAD_COEFF:
            r = e.dc(X, dY)
            close(host64(b.dC), r, what=f"dC[{j}]")


def run(batch, ops):
    ws = batch.workspace(ops)
    batch.run(ops, ws)
    torch.cuda.synchronize()


# ---------------------------------------------------------------------------
# the five workloads at oracle-friendly sizes (several tiles and a ragged tail)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("ops", [ffb.OP_FORWARD, ffb.OP_BACKWARD_DX, ffb.OP_GRAD_COEFF,
                                 ffb.OP_BACKWARD_DX | ffb.OP_GRAD_COEFF, ALL])
@pytest.mark.parametrize("unit", [True, False])
def test_single_256_fp32(ops, unit):
    b = AdapterBatch(wl.WORKLOADS["single_256_fp32"], DEV, unit_scale=unit, ops=ops)
    run(b, ops)
    check_batch(b, ops)


@pytest.mark.parametrize("kernel", ["tile", "tc", "tc2"])
@pytest.mark.parametrize("N", [37, 1, 4])
def test_roberta_base_all_matrices(N, kernel, monkeypatch):
    monkeypatch.setenv("FRAMEFB_KERNEL", kernel)
    b = AdapterBatch(wl.WORKLOADS["roberta_base_qv"], DEV, N=N, ops=ALL)
    run(b, ALL)
    check_batch(b, ALL)


@pytest.mark.parametrize("kernel", ["tile", "tc", "tc2"])
def test_vit_b16_mixed_shapes(kernel, monkeypatch):
    # many matrices of three shapes per launch: CTAs cross matrix boundaries
    monkeypatch.setenv("FRAMEFB_KERNEL", kernel)
    w = wl.WORKLOADS["vit_b16_merge"]
    b = AdapterBatch(w, DEV, N=23, ops=ALL)
    run(b, ALL)
    check_batch(b, ALL, js=[0, 3, 4, 5, 10, 11, 70, 71])


def test_llama2_shape_small_n():
    w = wl.WORKLOADS["llama2_7b_qkvo"]
    b = AdapterBatch(w, DEV, N=13, indices=[0, 5, 127], ops=ALL)
    run(b, ALL)
    check_batch(b, ALL)


@pytest.mark.parametrize("kernel", ["tc2", "tc", "tile"])
@pytest.mark.parametrize("ops", [ffb.OP_FORWARD, ffb.OP_BACKWARD_DX, ffb.OP_GRAD_COEFF,
                                 ffb.OP_BACKWARD_DX | ffb.OP_GRAD_COEFF, ALL])
def test_bf16_kernels_every_mode(kernel, ops, monkeypatch):
    # FRAMEFB_KERNEL selects the bf16 kernel: the one-phase-at-a-time
    # warp-MMA tile kernel, the one-token or the two-token tcgen05 kernel
    monkeypatch.setenv("FRAMEFB_KERNEL", kernel)
    w = wl.WORKLOADS["llama2_7b_qkvo"]
    b = AdapterBatch(w, DEV, N=13, indices=[0, 5], ops=ops)
    run(b, ops)
    check_batch(b, ops)


@pytest.mark.parametrize("kernel", ["tc2", "tile"])
@pytest.mark.parametrize("wname", ["roberta_blockdiag", "roberta_per_layer"])
def test_blockdiag_and_per_layer_supports(wname, kernel, monkeypatch):
    # supports inside the diagonal blocks of C, and a distinct support (and
    # plan) for every matrix of one launch
    monkeypatch.setenv("FRAMEFB_KERNEL", kernel)
    b = AdapterBatch(wl.WORKLOADS[wname], DEV, N=37, ops=ALL)
    run(b, ALL)
    check_batch(b, ALL)


@pytest.mark.parametrize("parts", ["1", "0"])
def test_llama3_zipf_nonsquare(parts, monkeypatch):
    # nnz = 8192 exceeds the register-resident chunk of the fused kernels and
    # d = 14336 their 128 groups: the plans' parts on the two-token tcgen05
    # kernel (FRAMEFB_PARTS=0: the split contraction path); X and dY shared
    # by the layer's matrices
    monkeypatch.setenv("FRAMEFB_PARTS", parts)
    w = wl.WORKLOADS["llama3_8b_all"]
    b = AdapterBatch(w, DEV, N=9, indices=list(range(7)), alias_inputs=True, ops=ALL)
    run(b, ALL)
    check_batch(b, ALL)


# ---------------------------------------------------------------------------
# semantics and edge cases
# ---------------------------------------------------------------------------
def test_entry_points_agree_with_fused():
    w = wl.WORKLOADS["roberta_base_qv"]
    fused = AdapterBatch(w, DEV, N=29, indices=[0, 1, 2], ops=ALL)
    run(fused, ALL)
    sep = AdapterBatch(w, DEV, N=29, indices=[0, 1, 2], ops=ALL)
    ws = sep.workspace(ALL)
    ffb.framefb_forward(sep.mats, sep.dtype_code, ws)
    ffb.framefb_backward_dx(sep.mats, sep.dtype_code, ws)
    ffb.framefb_grad_coeff(sep.mats, sep.dtype_code, ws)
    torch.cuda.synchronize()
    for a, c in zip(fused.bufs, sep.bufs):
        assert torch.equal(a.Y, c.Y) and torch.equal(a.dX, c.dX)
        assert torch.equal(a.dC, c.dC)        # deterministic reduction order


def test_accumulates_into_y_and_dx_fp32():
    w = wl.WORKLOADS["single_256_fp32"]
    b = AdapterBatch(w, DEV, N=11, y_init="random", ops=ALL)
    Y0, dX0 = host64(b.bufs[0].Y), host64(b.bufs[0].dX)
    run(b, ALL)
    e = Expect(b, 0)
    assert_f32(host64(b.bufs[0].Y), e.y(host64(b.bufs[0].X), Y0), what="Y")
    assert_f32(host64(b.bufs[0].dX), e.dx(host64(b.bufs[0].dY), dX0), what="dX")
    run(b, ffb.OP_FORWARD)             # a second call adds the delta again
    assert_f32(host64(b.bufs[0].Y), Y0 + 2 * (e.y(host64(b.bufs[0].X), Y0) - Y0), what="Y twice")


def test_deterministic_dc():
    w = wl.WORKLOADS["roberta_base_qv"]
    b = AdapterBatch(w, DEV, N=300, indices=[0, 1], ops=ffb.OP_GRAD_COEFF)
    run(b, ffb.OP_GRAD_COEFF)
    first = [x.dC.clone() for x in b.bufs]
    run(b, ffb.OP_GRAD_COEFF)
    for f, x in zip(first, b.bufs):
        assert torch.equal(f, x.dC)


def test_zero_tokens_gives_zero_dc_and_no_writes():
    w = wl.WORKLOADS["roberta_base_qv"]
    b = AdapterBatch(w, DEV, N=0, indices=[0], ops=ALL)
    run(b, ALL)
    assert torch.count_nonzero(b.bufs[0].dC) == 0


def test_empty_support_is_a_no_op():
    fin = ffb.Frame(256, 16, 16)
    dfin = fin.to_device(DEV)
    plan = ffb.Plan(fin, fin, np.zeros(0, np.int32), np.zeros(0, np.int32))
    pd = plan.to_device(DEV)
    X = torch.randn(10, 256, device=DEV, dtype=torch.bfloat16)
    Y = torch.randn(10, 256, device=DEV, dtype=torch.bfloat16)
    Y0 = Y.clone()
    m = ffb.make_mat(dfin, dfin, plan, pd, None, 1.0, 10, X=X, Y=Y)
    ffb.framefb_forward([m], ffb.FRAMEFB_BF16)
    torch.cuda.synchronize()
    assert torch.equal(Y, Y0)


@pytest.mark.parametrize("pad,off", [(64, 0), (8, 8)])
def test_strided_rows_and_untouched_padding(pad, off):
    # (64, 0): rows 32-byte aligned; (8, 8): rows only 16-byte aligned (leading
    # dimension = 8 mod 16 elements, region starting 16 bytes into the row)
    w = wl.WORKLOADS["roberta_base_qv"]
    N, n, m = 19, 768, 768
    src = AdapterBatch(w, DEV, N=N, indices=[0], ops=ALL)
    bb = src.bufs[0]
    Xp = torch.zeros(N, n + pad, device=DEV, dtype=torch.bfloat16)
    Xp[:, off:off + n] = bb.X
    dYp = torch.zeros(N + 2, m + pad, device=DEV, dtype=torch.bfloat16)
    dYp[:N, off:off + m] = bb.dY
    # padding holds sentinels; the active region starts at zero so that the
    # bf16 result is the delta itself
    Yp = torch.full((N + 2, m + pad), 3.0, device=DEV, dtype=torch.bfloat16)
    Yp[:N, off:off + m] = 0
    dXp = torch.full((N, n + pad), 5.0, device=DEV, dtype=torch.bfloat16)
    dXp[:, off:off + n] = 0
    dC = torch.zeros(w.nnz, device=DEV)
    mat = ffb.make_mat(src.dev_frames[n], src.dev_frames[m], src.plans[(m, n)], src.plan_dev[(m, n)], bb.c_val,
                       bb.scale, N, X=Xp[:, off:], dX=dXp[:, off:], dY=dYp[:, off:], Y=Yp[:, off:], dC=dC,
                       ldx=n + pad, ldy=m + pad)
    ws = ffb.workspace([mat], ALL, DEV)
    ffb.framefb_run([mat], ALL, ffb.FRAMEFB_BF16, ws)
    torch.cuda.synchronize()
    assert torch.all(Yp[:, off + m:] == 3.0) and torch.all(Yp[:, :off] == 3.0) and torch.all(Yp[N:, :] == 3.0)
    assert torch.all(dXp[:, off + n:] == 5.0) and torch.all(dXp[:, :off] == 5.0)
    e = Expect(src, 0)
    assert_bf16(host64(Yp[:N, off:off + m]), e.y(host64(bb.X), np.zeros((N, m))), what="Y strided")
    assert_bf16(host64(dXp[:, off:off + n]), e.dx(host64(bb.dY), np.zeros((N, n))), what="dX strided")
    assert_bf16(host64(dC), e.dc(host64(bb.X), host64(bb.dY)), what="dC strided")


def test_invalid_arguments_return_status():
    w = wl.WORKLOADS["roberta_base_qv"]
    b = AdapterBatch(w, DEV, N=8, indices=[0], ops=ALL)
    good = b.mats[0]
    bad = ffb.framefb_mat.from_buffer_copy(good)
    bad.X = good.X + 2                         # misaligned
    with pytest.raises(ffb.FramefbError) as e:
        ffb.framefb_run([bad], ALL, ffb.FRAMEFB_BF16, b.workspace(ALL))
    assert e.value.status == ffb.FRAMEFB_EINVAL
    with pytest.raises(ffb.FramefbError) as e:         # no workspace for dC
        ffb.framefb_run([good], ALL, ffb.FRAMEFB_BF16, None)
    assert e.value.status == ffb.FRAMEFB_EWORKSPACE
    bad = ffb.framefb_mat.from_buffer_copy(good)
    bad.n = 1024                               # frame / plan mismatch
    with pytest.raises(ffb.FramefbError) as e:
        ffb.framefb_run([bad], ffb.OP_FORWARD, ffb.FRAMEFB_BF16)
    assert e.value.status == ffb.FRAMEFB_EINVAL
    with pytest.raises(ffb.FramefbError) as e:
        ffb.framefb_run([good], 3 | 8, ffb.FRAMEFB_BF16)
    assert e.value.status == ffb.FRAMEFB_EINVAL


# ---------------------------------------------------------------------------
# merge
# ---------------------------------------------------------------------------
def _merge_case(wname, T=None):
    if wname == "single_256_fp32_many":          # 300 tenants x 8 out groups = 2400 work items
        import dataclasses
        w = dataclasses.replace(wl.WORKLOADS["single_256_fp32"], merge_tenants=300)
    else:
        w = wl.WORKLOADS[wname]
    m, n = w.merge_shape
    T = w.merge_tenants if T is None else T
    fin, fout = ffb.Frame(n, w.k, n // w.k), ffb.Frame(m, w.k, m // w.k)
    row, col, _, _ = ffb.framefb_support_build(m, n, w.nnz, w.support_seed, w.support_mode, w.zipf_s, w.k)
    plan = ffb.Plan(fin, fout, row, col)
    W0 = wl.w0_input(w, DEV)
    cv = wl.merge_c_values(w, DEV)[:T].contiguous()
    Wout = torch.full((T, m, n), float("nan"), device=DEV, dtype=W0.dtype)
    s = 200.0 / (m * n) ** 0.5
    ffb.framefb_merge(W0, fin.to_device(DEV), fout.to_device(DEV), plan, plan.to_device(DEV), cv, T, s, Wout)
    torch.cuda.synchronize()
    from oracle import adapter
    from tests.oracle_side import frame, oracle_support
    orow, ocol, _, _ = oracle_support(m, n, w.nnz, w.support_seed, w.support_mode, w.zipf_s, w.k)
    Cs = [adapter.dense_C(m, n, orow, ocol, host64(cv[t])) for t in range(T)]
    ref = adapter.merge(host64(W0), Cs, frame(n, w.k), frame(m, w.k), s)
    return host64(W0), host64(Wout), ref


def test_merge_fp32_delta_precision():
    W0, got, ref = _merge_case("single_256_fp32")
    for t in range(got.shape[0]):
        assert_f32(got[t] - W0, ref[t] - W0, what=f"dW[{t}]")


def test_merge_vit_64_tenants_bf16():
    W0, got, ref = _merge_case("vit_b16_merge")
    assert_bf16(got, ref, what="W_t")


# ---------------------------------------------------------------------------
# full size, in the launch configuration bench.py times
# ---------------------------------------------------------------------------
def test_llama2_full_size_bench_launch_sampled():
    """All 128 matrices x 8192 tokens in one fused launch; Y and dX checked on
    96 sampled token rows (rows are independent) and dC in full, for matrices
    of the first, a middle and the last layer."""
    w = wl.WORKLOADS["llama2_7b_qkvo"]
    b = AdapterBatch(w, DEV, ops=ALL)
    run(b, ALL)
    rng = np.random.default_rng(1)
    rows = np.unique(np.concatenate([[0, 1, w.N - 1], rng.choice(w.N, 93, replace=False)]))
    for j in (0, 66, 127):
        buf = b.bufs[j]
        e = Expect(b, j)
        X = host64(buf.X)
        dY = host64(buf.dY)
        assert_bf16(host64(buf.Y[torch.from_numpy(rows).to(DEV)]), e.y(X[rows], np.zeros((rows.size, 4096))),
                    what=f"Y[{j}] rows")
        assert_bf16(host64(buf.dX[torch.from_numpy(rows).to(DEV)]), e.dx(dY[rows], np.zeros((rows.size, 4096))),
                    what=f"dX[{j}] rows")
        assert_bf16(host64(buf.dC), e.dc(X, dY), what=f"dC[{j}]")
    del b
    torch.cuda.empty_cache()


# ---------------------------------------------------------------------------
# heavy-tailed supports on the default kernel, fp32 at size, many tenants
# ---------------------------------------------------------------------------
def _plan_header(plan):
    return np.frombuffer(plan.image()[:128].tobytes(), dtype=np.int32)


@pytest.mark.parametrize("nnz,N", [(1000, 37), (1000, 4096), (4096, 37)])
def test_zipf_rows_768_default_tcgen05_kernel(nnz, N):
    """Zipf(1.1) rows of C at 768 x 768: long runs of one row are split over
    chunks, so the row path writes overflow slots that the fix-up adds in
    (ovfZ 152 / 35 fix-ups at 1000 entries; the 4096-entry case fills every
    register chunk).  Runs on the default two-token tcgen05 kernel."""
    import dataclasses
    w = dataclasses.replace(wl.WORKLOADS["roberta_zipf"], nnz=nnz)
    b = AdapterBatch(w, DEV, N=N, ops=ALL)
    h = _plan_header(b.plans[(768, 768)])
    assert h[10] > 0 and h[12] > 0           # ovfZ, nfixZ: the fix-up path is exercised
    # packed units where the chunks hold at most 8 entries
    want = "tc2p_tile_kernel<7>" if max(h[8], h[9]) <= 8 else "tc2_tile_kernel<7>"
    assert ffb.framefb_kernel_names(b.mats, ALL, b.dtype_code) == [want]
    run(b, ALL)
    check_batch(b, ALL)


def test_fp32_large_n_with_sized_workspace():
    """fp32 activations at 4096 x 4096 and 8192 tokens with exactly the
    workspace framefb_workspace_size reports (the fp32 kernel's own grid)."""
    w = wl.Workload("fp32_4096", (wl.MatSpec("w", 4096, 4096),), N=8192, nnz=4096, dtype="f32", c_std=0.01)
    b = AdapterBatch(w, DEV, ops=ALL)
    need = ffb.framefb_workspace_size(b.mats, ALL)
    assert need > 0
    ws = torch.empty(need, dtype=torch.uint8, device=DEV)
    assert ffb.framefb_kernel_names(b.mats, ALL, b.dtype_code) == ["fft_tile_kernel<7>"]
    ffb.framefb_run(b.mats, ALL, b.dtype_code, ws)
    torch.cuda.synchronize()
    rows = np.unique(np.concatenate([[0, w.N - 1], np.random.default_rng(3).choice(w.N, 62, replace=False)]))
    buf, e = b.bufs[0], Expect(b, 0)
    X, dY = host64(buf.X), host64(buf.dY)
    sel = torch.from_numpy(rows).to(DEV)
    assert_f32(host64(buf.Y[sel]), e.y(X[rows], np.zeros((rows.size, 4096))), what="Y rows")
    assert_f32(host64(buf.dX[sel]), e.dx(dY[rows], np.zeros((rows.size, 4096))), what="dX rows")
    assert_f32(host64(buf.dC), e.dc(X, dY), what="dC")


def test_merge_many_tenants_grid_stride():
    """More (out group, tenant) items than resident CTAs: every item is taken
    by the grid-stride loop exactly once."""
    W0, got, ref = _merge_case("single_256_fp32_many")
    for t in (0, 1, 77, got.shape[0] - 1):
        assert_f32(got[t] - W0, ref[t] - W0, what=f"dW[{t}]")


# ---------------------------------------------------------------------------
# plans the fused tcgen05 kernels do not take: the split contraction path
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("ops", [ffb.OP_FORWARD, ffb.OP_BACKWARD_DX, ffb.OP_GRAD_COEFF,
                                 ffb.OP_BACKWARD_DX | ffb.OP_GRAD_COEFF, ALL])
def test_llama3_shapes_run_as_parts(ops):
    """LLaMA-3 shapes (Zipf support with 32 entries per plan column, d up to
    14336 = 448 groups) run as their plans' parts on the two-token tcgen05
    kernel, parts that write the same features in successive launches, for
    every op mask; Y and dX accumulate the parts' contributions.  The down
    projection (14336 inputs) has no parts and runs on the split path."""
    w = wl.WORKLOADS["llama3_8b_all"]
    b = AdapterBatch(w, DEV, N=45, indices=list(range(7)), ops=ops)
    for k in set(b.keys):
        assert bool(b.plans[k].parts()) == (k[1] <= 4096), k   # key (m, n)
    names = ffb.framefb_kernel_names(b.mats, ops, b.dtype_code)
    assert f"tc2_tile_kernel<{ops}>" in names and any(x.startswith("dense_") for x in names)
    run(b, ops)
    check_batch(b, ops)
    if ops & (ffb.OP_FORWARD | ffb.OP_BACKWARD_DX):
        y1 = [(x.Y.float().clone() if x.Y is not None else None, x.dX.float().clone() if x.dX is not None else None)
              for x in b.bufs]
        run(b, ops)
        # doubled within the bf16 bar: the parts round once each
        for (ya, xa), x in zip(y1, b.bufs):
            for on, got, once in ((ops & ffb.OP_FORWARD, x.Y, ya), (ops & ffb.OP_BACKWARD_DX, x.dX, xa)):
                if on:
                    rms = float(once.pow(2).mean().sqrt())
                    torch.testing.assert_close(got.float(), 2 * once, rtol=2e-2, atol=2e-2 * 2 * rms)


def test_llama3_shapes_take_the_split_path(monkeypatch):
    """With FRAMEFB_PARTS=0 the LLaMA-3 shapes run as grouped K = 32
    contractions around the SpMM; with FRAMEFB_KERNEL=tile the same call runs
    on the warp-MMA kernel, and both agree with the oracle."""
    monkeypatch.setenv("FRAMEFB_PARTS", "0")
    w = wl.WORKLOADS["llama3_8b_all"]
    b = AdapterBatch(w, DEV, N=45, indices=list(range(7)), ops=ALL)
    names = ffb.framefb_kernel_names(b.mats, ALL, b.dtype_code)
    assert "dense_gemm_kernel<bf16_hilo><grouped>" in names and "mma_tile_kernel<7>" not in names
    run(b, ALL)
    check_batch(b, ALL)


def test_llama3_shapes_on_the_warp_mma_kernel(monkeypatch):
    monkeypatch.setenv("FRAMEFB_KERNEL", "tile")
    w = wl.WORKLOADS["llama3_8b_all"]
    b = AdapterBatch(w, DEV, N=21, indices=[1, 4, 6], ops=ALL)
    assert ffb.framefb_kernel_names(b.mats, ALL, b.dtype_code) == ["mma_tile_kernel<7>"]
    run(b, ALL)
    check_batch(b, ALL)


@pytest.mark.parametrize("parts", ["1", "0"])
def test_padded_rows_of_large_plans(parts, monkeypatch):
    """Padded rows (a leading dimension above the features) of a large plan:
    its parts on the two-token tcgen05 kernel take strided rows; without parts
    the split path (which views rows as [tokens * groups][32]) does not, and
    the plan stays on the fused warp-MMA kernel."""
    monkeypatch.setenv("FRAMEFB_PARTS", parts)
    w = wl.WORKLOADS["llama3_8b_all"]
    N, pad = 17, 64
    src = AdapterBatch(w, DEV, N=N, indices=[1], ops=ALL)   # k: 4096 -> 1024
    bb = src.bufs[0]
    n, m = bb.spec.n, bb.spec.m
    Xp = torch.zeros(N, n + pad, device=DEV, dtype=torch.bfloat16)
    Xp[:, :n] = bb.X
    dYp = torch.zeros(N, m + pad, device=DEV, dtype=torch.bfloat16)
    dYp[:, :m] = bb.dY
    Yp = torch.zeros(N, m + pad, device=DEV, dtype=torch.bfloat16)
    dXp = torch.zeros(N, n + pad, device=DEV, dtype=torch.bfloat16)
    dC = torch.zeros(w.nnz, device=DEV)
    key = src.keys[0]
    mat = ffb.make_mat(src.dev_frames[n], src.dev_frames[m], src.plans[key], src.plan_dev[key], bb.c_val, bb.scale, N,
                       X=Xp, dX=dXp, dY=dYp, Y=Yp, dC=dC, ldx=n + pad, ldy=m + pad)
    assert ffb.framefb_kernel_names([mat], ALL, ffb.FRAMEFB_BF16) == (["tc2_tile_kernel<7>"] if parts == "1"
                                                                       else ["mma_tile_kernel<7>"])
    ffb.framefb_run([mat], ALL, ffb.FRAMEFB_BF16, ffb.workspace([mat], ALL, DEV))
    torch.cuda.synchronize()
    e = Expect(src, 0)
    assert_bf16(host64(Yp[:, :m]), e.y(host64(bb.X), np.zeros((N, m))), what="Y padded")
    assert_bf16(host64(dXp[:, :n]), e.dx(host64(bb.dY), np.zeros((N, n))), what="dX padded")
    assert_bf16(host64(dC), e.dc(host64(bb.X), host64(bb.dY)), what="dC padded")
