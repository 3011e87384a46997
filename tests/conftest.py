import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: full-size parity case")


@pytest.fixture(autouse=True)
def _no_wait_timeouts(request):
    """GPU tests: no bounded wait of a kernel may give up during the test
    (a CTA that gives up stops early and leaves its results incomplete)."""
    if request.node.get_closest_marker("gpu") is None:
        yield
        return
    import torch
    if not torch.cuda.is_available():
        yield
        return
    from paper_2608_26430_gb300 import framefb as ffb
    try:
        before = ffb.framefb_wait_timeouts()
    except Exception:
        before = None  # the library is built by the test module's own fixture
    yield
    if before is None:
        return
    assert ffb.framefb_wait_timeouts() == before, "a kernel's bounded wait gave up during this test"
