"""Full-size GPU parity of the evaluation workloads, in the launch
configuration bench.py times (one framefb_run over all the workload's
matrices at its full token count), against the fp64 oracle.

Rows of Y and dX are independent, so they are checked on sampled token rows
(always including the first and the last); dC sums over every token and is
checked in full.  Tolerances are the bf16 bar of test_gpu_parity.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2608_26430_gb300 import framefb as ffb
from paper_2608_26430_gb300 import workloads as wl
from paper_2608_26430_gb300.batch import AdapterBatch
from tests.oracle_side import Expect, assert_bf16, host64

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

DEV = "cuda:0"
ALL = ffb.OP_FORWARD | ffb.OP_BACKWARD_DX | ffb.OP_GRAD_COEFF


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_26430_gb300.build import build
    build()
    ffb.lib()


def sampled_rows(N, k, seed):
    rng = np.random.default_rng(seed)
    return np.unique(np.concatenate([[0, 1, N - 1], rng.choice(N, k, replace=False)]))


def check_sampled(b, js, rows):
    sel = torch.from_numpy(rows).to(DEV)
    for j in js:
        buf, e = b.bufs[j], Expect(b, j)
        X, dY = host64(buf.X), host64(buf.dY)
        assert_bf16(host64(buf.Y[sel]), e.y(X[rows], np.zeros((rows.size, buf.spec.m))), what=f"Y[{j}] rows")
        assert_bf16(host64(buf.dX[sel]), e.dx(dY[rows], np.zeros((rows.size, buf.spec.n))), what=f"dX[{j}] rows")
        assert_bf16(host64(buf.dC), e.dc(X, dY), what=f"dC[{j}]")


def run_full(b):
    ws = b.workspace(ALL)
    b.run(ALL, ws)
    torch.cuda.synchronize()


def test_roberta_full_size_every_matrix():
    """24 q/v matrices of 768 x 768 at 4096 tokens: every row of every matrix."""
    w = wl.WORKLOADS["roberta_base_qv"]
    b = AdapterBatch(w, DEV, ops=ALL)
    assert ffb.framefb_kernel_names(b.mats, ALL, b.dtype_code) == ["tc2p_tile_kernel<7>"]
    run_full(b)
    check_sampled(b, range(len(b.bufs)), np.arange(w.N))


def test_vit_full_size_sampled():
    """72 matrices of three shapes at 64 x 197 tokens (a ragged last token
    pair); the first and the last layer's q, fc1, fc2 and a middle layer."""
    w = wl.WORKLOADS["vit_b16_merge"]
    b = AdapterBatch(w, DEV, ops=ALL)
    run_full(b)
    check_sampled(b, [0, 4, 5, 33, 66, 70, 71], sampled_rows(w.N, 125, 5))


def test_llama3_full_layer_sampled():
    """One full LLaMA-3-8B-shaped layer (q, GQA k/v, o, gate, up, down:
    d in {1024, 4096, 14336}) at 16384 tokens with the Zipf(1.1) support,
    every matrix checked."""
    w = wl.WORKLOADS["llama3_8b_all"]
    b = AdapterBatch(w, DEV, indices=list(range(7)), ops=ALL)
    run_full(b)
    check_sampled(b, range(7), sampled_rows(w.N, 93, 7))
    del b
    torch.cuda.empty_cache()
