"""Adaptive segmented LUTs (host side).

The paper's nonlinear primitives split the input domain [tau_0, tau_Nseg]
into N_seg segments with boundaries tau_j (logarithmically spaced for 1/x and
1/sqrt(x), uniformly for SiLU/GELU), give each segment its own table of N_br
equal intervals, and approximate f on interval i of segment s by a line
a_si x + b_si (Segmented LUT Evaluation, "Adaptive LUT Construction").  The
online lookup finds the segment S (comparisons with the boundaries), the
local interval I = floor((x - tau_S)/(tau_{S+1} - tau_S) N_br) and returns
a_SI x + b_SI ("Online Lookup Evaluation", Steps 1-3).  The encrypted
protocol packs the same numbers into plaintext polynomials (Cryptographic
Lookup Protocol): p(X), q(X) for the interval index and a_s(X), b_s(X) for
the candidate values.

Each interval's line interpolates f at the interval's two Chebyshev nodes
c +- (h/2) cos(pi/4) (c its centre, h its width): the near-minimax linear
fit, and the one that reproduces the paper's printed coefficients.
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

FUNCTIONS = {
    "reciprocal": lambda x: 1.0 / x,
    "rsqrt": lambda x: 1.0 / math.sqrt(x),
    "gelu": lambda x: 0.5 * x * (1.0 + math.erf(x / math.sqrt(2.0))),
    "silu": lambda x: x / (1.0 + math.exp(-x)),
    "exp": math.exp,
}


def boundaries(lo: float, hi: float, n_seg: int, spacing: str) -> list:
    """tau_0 = lo < ... < tau_Nseg = hi, uniform or logarithmic (lo > 0)."""
    if spacing == "uniform":
        return [lo + (hi - lo) * j / n_seg for j in range(n_seg + 1)]
    if spacing == "log":
        if lo <= 0:
            raise ValueError("logarithmic boundaries need lo > 0")
        return [lo * (hi / lo) ** (j / n_seg) for j in range(n_seg + 1)]
    raise ValueError(spacing)


@dataclass
class SegmentedLUT:
    tau: list          # N_seg + 1 boundaries
    n_br: int          # intervals per segment
    a: np.ndarray      # [N_seg][N_br] slopes
    b: np.ndarray      # [N_seg][N_br] offsets

    @property
    def n_seg(self) -> int:
        return len(self.tau) - 1


def build(f, tau, n_br: int) -> SegmentedLUT:
    """Per-interval lines through f at the two Chebyshev nodes."""
    n_seg = len(tau) - 1
    a = np.zeros((n_seg, n_br))
    b = np.zeros((n_seg, n_br))
    r = math.cos(math.pi / 4) / 2
    for s in range(n_seg):
        h = (tau[s + 1] - tau[s]) / n_br
        for i in range(n_br):
            c = tau[s] + (i + 0.5) * h
            x1, x2 = c - r * h, c + r * h
            y1, y2 = f(x1), f(x2)
            a[s, i] = (y2 - y1) / (x2 - x1)
            b[s, i] = y1 - a[s, i] * x1
    return SegmentedLUT(list(tau), n_br, a, b)


def segment_index(lut: SegmentedLUT, x: float) -> int:
    """Step 1: S = sum_{j=1}^{N_seg-1} [x >= tau_j]."""
    return sum(1 for j in range(1, lut.n_seg) if x >= lut.tau[j])


def interval_index(lut: SegmentedLUT, x: float, s: int) -> int:
    """Step 2: I = floor((x - tau_S) / (tau_{S+1} - tau_S) N_br), kept in the table."""
    i = math.floor((x - lut.tau[s]) / (lut.tau[s + 1] - lut.tau[s]) * lut.n_br)
    return min(max(i, 0), lut.n_br - 1)


def lookup(lut: SegmentedLUT, x: float) -> float:
    """Step 3: a_SI x + b_SI."""
    s = segment_index(lut, x)
    i = interval_index(lut, x, s)
    return float(lut.a[s, i] * x + lut.b[s, i])


def index_polynomials(lut: SegmentedLUT):
    """Coefficients of p(X) = sum_s N_br/(tau_{s+1}-tau_s) X^s and
    q(X) = sum_s -tau_s N_br/(tau_{s+1}-tau_s) X^s: p x + q holds each
    segment's candidate interval index at coefficient s."""
    w = np.array([lut.n_br / (lut.tau[s + 1] - lut.tau[s]) for s in range(lut.n_seg)])
    return w, -np.array(lut.tau[:-1]) * w


def value_polynomials(lut: SegmentedLUT, s: int):
    """Coefficients of a_s(X) = sum_i a_si X^i and b_s(X) = sum_i b_si X^i."""
    return lut.a[s].copy(), lut.b[s].copy()
