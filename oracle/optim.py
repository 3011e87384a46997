"""Oracle: the optimiser step on the adapter coefficients, fp64.

Test infrastructure only (see ``oracle/__init__``).

The paper trains the coefficient values with AdamW under a linear
learning-rate schedule with warmup (Appendix "Hyperparameters used for the
experiments": the GLUE, image-classification and instruction-tuning tables
give the optimiser, the schedule, the adapter learning rate and the warmup
ratio).  The tables give neither the moment decay rates, nor epsilon, nor the
weight decay; the reading taken here is the defaults of the stock PyTorch
optimiser the paper's implementation runs on (Sec. 4.7): beta1 = 0.9,
beta2 = 0.999, eps = 1e-8, weight decay = 0.01.

AdamW (Adam with decoupled weight decay, Loshchilov and Hutter), step t >= 1
on parameters p with gradient g and moments m, v (zero before step 1):

    p <- p * (1 - lr * wd)                       decoupled weight decay
    m <- beta1 * m + (1 - beta1) * g             first moment
    v <- beta2 * v + (1 - beta2) * g^2           second moment
    p <- p - lr * (m / (1 - beta1^t)) / (sqrt(v / (1 - beta2^t)) + eps)

Linear schedule with warmup over `total` steps, `warmup` of them warming up:
the learning rate of the step with 0-based index i is
    lr_max * i / warmup                          for i < warmup
    lr_max * max(0, (total - i) / (total - warmup))   otherwise.
"""
from __future__ import annotations

import numpy as np

DEFAULTS = dict(beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)


def adamw_step(p, g, m, v, t: int, lr: float, beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8,
               weight_decay: float = 0.01):
    """One AdamW step t (1-based); returns the new (p, m, v) as fp64 arrays."""
    if t < 1:
        raise ValueError("the step count starts at 1")
    p = np.asarray(p, dtype=np.float64) * (1.0 - lr * weight_decay)
    g = np.asarray(g, dtype=np.float64)
    m = beta1 * np.asarray(m, dtype=np.float64) + (1.0 - beta1) * g
    v = beta2 * np.asarray(v, dtype=np.float64) + (1.0 - beta2) * g * g
    m_hat = m / (1.0 - beta1 ** t)
    v_hat = v / (1.0 - beta2 ** t)
    p = p - lr * m_hat / (np.sqrt(v_hat) + eps)
    return p, m, v


def linear_warmup_lr(i: int, total: int, warmup: int, lr_max: float) -> float:
    """Learning rate of the step with 0-based index i."""
    if i < warmup:
        return lr_max * i / warmup
    if total <= warmup:
        return 0.0
    return lr_max * max(0.0, (total - i) / (total - warmup))
