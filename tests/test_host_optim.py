"""CPU tests of the host side of the widening entry points: the optimiser's
learning-rate schedule against the oracle, and the argument checks of the
optimiser step and of the mixed-tenant forward, which return before any
device work."""
import ctypes as ct

import pytest

from oracle import optim
from paper_2608_26430_gb300 import framefb as ffb


@pytest.fixture(scope="module", autouse=True)
def built_library():
    from paper_2608_26430_gb300.build import build
    build()


@pytest.mark.parametrize("total,warmup,lr", [(100, 6, 0.33), (17, 0, 0.12), (10, 10, 0.1), (1000, 30, 3e-3)])
def test_linear_warmup_schedule_matches_oracle(total, warmup, lr):
    for i in range(0, total + 5):
        got = ffb.framefb_linear_warmup_lr(i, total, warmup, lr)
        assert got == pytest.approx(optim.linear_warmup_lr(i, total, warmup, lr), rel=1e-15, abs=0.0)
    assert ffb.framefb_linear_warmup_lr(-1, total, warmup, lr) == 0.0


def _adamw(p, g, m, v, n, hp, step):
    return ffb.lib().framefb_adamw(p, g, m, v, n, hp, step, None)


def test_adamw_argument_checks_before_any_device_work():
    ok = ffb.framefb_adamw_params(0.1, 0.9, 0.999, 1e-8, 0.01)
    P = 4096  # an aligned stand-in address; none of these calls reaches the device
    assert _adamw(P, P + 4096, P + 8192, P + 12288, 0, ct.byref(ok), 1) == ffb.FRAMEFB_OK  # n == 0: no-op
    assert _adamw(P, P, P, P, -1, ct.byref(ok), 1) == ffb.FRAMEFB_EINVAL
    assert _adamw(P, P, P, P, 8, ct.byref(ok), 0) == ffb.FRAMEFB_EINVAL
    assert _adamw(P, P, P, P, 8, None, 1) == ffb.FRAMEFB_EINVAL
    assert _adamw(None, P, P, P, 8, ct.byref(ok), 1) == ffb.FRAMEFB_EINVAL
    assert _adamw(P + 2, P, P, P, 8, ct.byref(ok), 1) == ffb.FRAMEFB_EINVAL  # not 4-byte aligned
    for bad in [(-0.1, 0.9, 0.999, 1e-8, 0.0), (0.1, 1.0, 0.999, 1e-8, 0.0), (0.1, 0.9, -0.5, 1e-8, 0.0),
                (0.1, 0.9, 0.999, 0.0, 0.0), (0.1, 0.9, 0.999, 1e-8, -1.0), (float("nan"), 0.9, 0.999, 1e-8, 0.0)]:
        hp = ffb.framefb_adamw_params(*bad)
        assert _adamw(P, P, P, P, 8, ct.byref(hp), 1) == ffb.FRAMEFB_EINVAL, bad


def test_tenant_segment_tables_are_checked_before_any_device_work():
    from paper_2608_26430_gb300 import workloads as wl
    fin = ffb.Frame(768, 16, 48)
    row, col, _, _ = ffb.framefb_support_build(768, 768, 100, 1, wl.UNIFORM, 1.1, 16)
    plan = ffb.Plan(fin, fin, row, col)
    mat = ffb.framefb_mat()
    mat.N, mat.n, mat.m, mat.plan = 10, 768, 768, plan.handle.value
    arr = (ffb.framefb_mat * 1)(mat)

    def call(starts, tenants, ntenants=2, n=1):
        s = (ct.c_int32 * len(starts))(*starts)
        t = (ct.c_int32 * max(len(tenants), 1))(*tenants)
        return ffb.lib().framefb_forward_tenants(arr, n, ffb.FRAMEFB_BF16, s, t, len(tenants), ntenants, None)

    assert call([1, 10], [0]) == ffb.FRAMEFB_EINVAL          # does not start at token 0
    assert call([0, 6, 4, 10], [0, 1, 0]) == ffb.FRAMEFB_EINVAL  # decreasing
    assert call([0, 5, 10], [0, 2]) == ffb.FRAMEFB_EINVAL      # tenant out of range
    assert call([0, 5, 9], [0, 1]) == ffb.FRAMEFB_EINVAL       # ends before the matrices' N
    assert call([0, 10], [0], ntenants=0) == ffb.FRAMEFB_EINVAL
    assert call([0, 10], [0], n=0) == ffb.FRAMEFB_OK            # no matrices: nothing to do
