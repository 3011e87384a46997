"""Pins of the oracle's optimiser step: the library AdamW of PyTorch (CPU,
fp64) over several steps, the closed form of the first step, pure weight
decay, and the schedule's corner values."""
import numpy as np
import pytest

from oracle import optim


def test_adamw_matches_the_library_optimizer_over_steps():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(11)
    n, steps, total, warmup, lr_max = 257, 6, 20, 3, 0.12
    p0 = rng.standard_normal(n) * 0.01
    grads = [rng.standard_normal(n) * 10.0 ** rng.uniform(-3, 1) for _ in range(steps)]
    tp = torch.tensor(p0, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([tp], lr=lr_max, betas=(0.9, 0.999), eps=1e-8, weight_decay=0.01)
    p, m, v = p0.copy(), np.zeros(n), np.zeros(n)
    for i, g in enumerate(grads):
        lr = optim.linear_warmup_lr(i + 1, total, warmup, lr_max)  # step 0 would have lr 0
        for grp in opt.param_groups:
            grp["lr"] = lr
        tp.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        p, m, v = optim.adamw_step(p, g, m, v, i + 1, lr, **optim.DEFAULTS)
        np.testing.assert_allclose(p, tp.detach().numpy(), rtol=1e-13, atol=1e-16)
        st = opt.state[tp]
        np.testing.assert_allclose(m, st["exp_avg"].numpy(), rtol=1e-13, atol=0)
        np.testing.assert_allclose(v, st["exp_avg_sq"].numpy(), rtol=1e-13, atol=0)


def test_first_step_closed_form():
    # with zero moments the bias-corrected moments are g and g^2: the update is lr g / (|g| + eps)
    g = np.array([3.0, -0.5, 1e-9, 0.0, -2e-12])
    p0 = np.array([1.0, -2.0, 0.5, 0.25, 4.0])
    lr, eps = 0.3, 1e-8
    p, m, v = optim.adamw_step(p0, g, np.zeros(5), np.zeros(5), 1, lr, 0.9, 0.999, eps, 0.0)
    np.testing.assert_allclose(p, p0 - lr * g / (np.abs(g) + eps), rtol=1e-14)
    np.testing.assert_allclose(m, 0.1 * g, rtol=1e-15)
    np.testing.assert_allclose(v, 0.001 * g * g, rtol=1e-12)


def test_zero_gradient_is_pure_decay():
    p = np.array([1.5, -3.0, 0.0, 7.0])
    m = v = np.zeros(4)
    lr, wd = 0.1, 0.05
    for t in range(1, 6):
        p, m, v = optim.adamw_step(p, np.zeros(4), m, v, t, lr, 0.9, 0.999, 1e-8, wd)
    np.testing.assert_allclose(p, np.array([1.5, -3.0, 0.0, 7.0]) * (1 - lr * wd) ** 5, rtol=1e-15)


def test_linear_warmup_schedule_corners():
    lr = 0.33
    assert optim.linear_warmup_lr(0, 100, 6, lr) == 0.0
    assert optim.linear_warmup_lr(3, 100, 6, lr) == pytest.approx(lr / 2, rel=1e-15)
    assert optim.linear_warmup_lr(6, 100, 6, lr) == pytest.approx(lr, rel=1e-15)
    assert optim.linear_warmup_lr(53, 100, 6, lr) == pytest.approx(lr / 2, rel=1e-15)
    assert optim.linear_warmup_lr(100, 100, 6, lr) == 0.0
    assert optim.linear_warmup_lr(150, 100, 6, lr) == 0.0
    assert optim.linear_warmup_lr(0, 10, 0, lr) == pytest.approx(lr, rel=1e-15)


def test_step_count_starts_at_one():
    with pytest.raises(ValueError):
        optim.adamw_step(np.zeros(2), np.zeros(2), np.zeros(2), np.zeros(2), 0, 0.1)
