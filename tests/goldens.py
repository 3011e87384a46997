"""Readers for the worked-example fixtures under tests/golden/ (no arithmetic of the method)."""
import cmath
import math
import os
import re

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")

_TERM = re.compile(r"^(sqrt\((\d+)\)|\d+)$")


def _term(tok: str) -> float:
    m = _TERM.match(tok)
    if not m:
        raise ValueError(f"bad term {tok!r}")
    return math.sqrt(int(m.group(2))) if m.group(2) else float(tok)


def parse_coef(expr: str) -> float:
    """'-sqrt(2)/sqrt(3)' -> float; products with '*', one optional '/'."""
    sign = -1.0 if expr.startswith("-") else 1.0
    expr = expr.lstrip("-")
    num, _, den = expr.partition("/")
    val = 1.0
    for t in num.split("*"):
        val *= _term(t)
    if den:
        for t in den.split("*"):
            val /= _term(t)
    return sign * val


def _rows(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


def load_real_matrix(name) -> np.ndarray:
    return np.array([[parse_coef(t) for t in r] for r in _rows(name)], dtype=np.float64)


def load_omega_matrix(name, k) -> np.ndarray:
    omega = cmath.exp(2j * math.pi / k)
    out = []
    for r in _rows(name):
        row = []
        for t in r:
            if t == "0":
                row.append(0j)
            else:
                c, _, p = t.partition("@")
                row.append(parse_coef(c) * omega ** int(p))
        out.append(row)
    return np.array(out, dtype=np.complex128)
