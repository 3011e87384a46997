"""GPU parity of the optimiser step (framefb_adamw) against the fp64 oracle,
and a short training loop: fused forward/backward, then AdamW on the
coefficients of all matrices in one call, then the next forward with the
updated coefficients."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import optim
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


def _f32(a):
    return torch.tensor(np.asarray(a, np.float32), device=DEV)


def _as_f32(hp):
    # the library takes its hyperparameters as fp32: the oracle gets the same values
    return {k: float(np.float32(x)) for k, x in hp.items()}


@pytest.mark.parametrize("n,offset", [(4 * 1000 + 3, 0), (4 * 1000 + 3, 1), (1, 0), (64 * 4096, 0)])
def test_adamw_matches_oracle_over_steps(n, offset):
    # offset 1: arrays start 4 bytes into an allocation (the single-value path)
    rng = np.random.default_rng(n + offset)
    hp = dict(beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)
    p0 = (rng.standard_normal(n) * 0.01).astype(np.float32)
    buf = {k: torch.zeros(n + offset, dtype=torch.float32, device=DEV) for k in ("p", "g", "m", "v")}
    dev = {k: b[offset:] for k, b in buf.items()}
    dev["p"].copy_(_f32(p0))
    p, m, v = p0.astype(np.float64), np.zeros(n), np.zeros(n)
    total, warmup, lr_max = 50, 3, 0.12
    for t in range(1, 6):
        g = (rng.standard_normal(n) * 10.0 ** rng.uniform(-4, 1)).astype(np.float32)
        dev["g"].copy_(_f32(g))
        lr = optim.linear_warmup_lr(t, total, warmup, lr_max)
        ffb.framefb_adamw(dev["p"], dev["g"], dev["m"], dev["v"], t, lr, **hp)
        p, m, v = optim.adamw_step(p, g, m, v, t, float(np.float32(lr)), **_as_f32(hp))
    torch.cuda.synchronize()
    assert_f32(host64(dev["p"]), p, what="param")
    assert_f32(host64(dev["m"]), m, what="m")
    assert_f32(host64(dev["v"]), v, what="v")


def test_adamw_empty_and_invalid():
    x = torch.zeros(8, dtype=torch.float32, device=DEV)
    ffb.framefb_adamw(x, x, x, x, 1, 0.1, n=0)  # no-op
    with pytest.raises(ffb.FramefbError) as e:
        ffb.framefb_adamw(x, x, x, x, 0, 0.1)
    assert e.value.status == ffb.FRAMEFB_EINVAL


def test_training_loop_through_the_c_abi():
    w = wl.WORKLOADS["roberta_base_qv"]
    idx = [0, 1, 7]
    b = AdapterBatch(w, DEV, N=96, indices=idx, ops=ALL)
    ws = b.workspace(ALL)
    L, nnz = b.C.shape
    m = torch.zeros_like(b.C)
    v = torch.zeros_like(b.C)
    ex = [Expect(b, j) for j in range(len(idx))]
    X = [host64(bb.X) for bb in b.bufs]
    dY = [host64(bb.dY) for bb in b.bufs]
    dc_ref = np.stack([ex[j].dc(X[j], dY[j]) for j in range(L)])
    # eps well above the gradient's rounding error keeps the update a smooth
    # function of the gradient (|du/dg| <= 1/eps), so the two trajectories
    # stay within lr * (gradient error) / eps of each other
    hp = dict(beta1=0.9, beta2=0.999, eps=1e-2 * float(np.sqrt(np.mean(dc_ref ** 2))), weight_decay=0.01)
    c, mo, vo = np.stack([e.c for e in ex]), np.zeros((L, nnz)), np.zeros((L, nnz))
    total, warmup, lr_max = 10, 2, 0.05
    for t in range(1, 4):
        for bb in b.bufs:
            bb.Y.zero_()
            bb.dX.zero_()
        b.run(ALL, ws)
        lr = optim.linear_warmup_lr(t, total, warmup, lr_max)
        ffb.framefb_adamw(b.C, b.dC, m, v, t, lr, **hp)
        c, mo, vo = optim.adamw_step(c, dc_ref, mo, vo, t, float(np.float32(lr)), **_as_f32(hp))
    torch.cuda.synchronize()
    steps_lr = sum(optim.linear_warmup_lr(t, total, warmup, lr_max) for t in range(1, 4))
    got = host64(b.C)
    assert np.max(np.abs(got - c)) <= 2e-3 * steps_lr, np.max(np.abs(got - c))
    assert np.max(np.abs(got - np.stack([e.c for e in ex]))) > 0.5 * steps_lr  # the coefficients moved
    # the next forward pass sees the updated coefficients
    for bb in b.bufs:
        bb.Y.zero_()
    b.run(ffb.OP_FORWARD, ws)
    torch.cuda.synchronize()
    from oracle import adapter
    for j, bb in enumerate(b.bufs):
        e = ex[j]
        C_new = np.zeros_like(e.C)
        C_new[e.row, e.col] = c[j]
        y_ref = adapter.forward(X[j], np.zeros((X[j].shape[0], bb.spec.m)), e.Pin, e.Pout, C_new, e.scale)
        assert_bf16(host64(bb.Y), y_ref, what=f"Y after training, matrix {j}")
