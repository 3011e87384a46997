"""The workspace-free entry point framefb_run_static_ws.

It serves callers that cannot allocate device memory where they call the
library; its dC partial sums live in a static device array of the library.
Checked here through the C ABI against framefb_run with a caller workspace,
on two calls in a row (Y and dX accumulate, dC is overwritten), plus the
size limit.  This file is collected last on purpose.
"""
import pytest

torch = pytest.importorskip("torch")

from paper_2608_26430_gb300 import framefb as ffb
from paper_2608_26430_gb300 import workloads as wl
from paper_2608_26430_gb300.batch import AdapterBatch
from tests.oracle_side import assert_bf16, host64

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


def test_static_workspace_matches_caller_workspace_twice():
    w = wl.WORKLOADS["vit_b16_merge"]
    idx = [0, 4, 5, 10]                      # 768x768, 768->3072, 3072->768 shapes
    ref = AdapterBatch(w, DEV, N=77, indices=idx, ops=ALL)
    got = AdapterBatch(w, DEV, N=77, indices=idx, ops=ALL)
    ws = ref.workspace(ALL)
    for call in range(2):
        ffb.framefb_run(ref.mats, ALL, ref.dtype_code, ws)
        ffb.framefb_run_static_ws(got.mats, ALL, got.dtype_code)
        torch.cuda.synchronize()
        # the same kernels on the same inputs: bit-equal results, and both
        # within the bf16 bar of each other
        for a, b in zip(ref.bufs, got.bufs):
            for x, y, nm in ((a.Y, b.Y, "Y"), (a.dX, b.dX, "dX"), (a.dC, b.dC, "dC")):
                assert torch.equal(x, y), f"call {call} {nm}: static and caller workspace differ"
                assert_bf16(host64(y), host64(x), what=f"call {call} {nm}")


def test_static_workspace_rejects_oversized_calls():
    # rho = 2 frames at 768 over 4096 tokens: the contraction path keeps the
    # frame coefficients of the tokens in its workspace (about 50 MB), more
    # than the 8 MiB array
    w = wl.WORKLOADS["roberta_rho2"]
    b = AdapterBatch(w, DEV, indices=[0], ops=ALL)
    assert ffb.framefb_workspace_size(b.mats, ALL) > ffb.STATIC_WS_BYTES
    with pytest.raises(ffb.FramefbError) as e:
        ffb.framefb_run_static_ws(b.mats, ALL, b.dtype_code)
    assert e.value.status == ffb.FRAMEFB_EWORKSPACE
