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

``encode`` turns a table into the integer polynomials the encrypted lookup
(``rosetta_segmented_lookup_batch``) takes.  A "coefficient" selected by an
encrypted index is a box of N/K ring coefficients (K = N_seg or N_br), laid
out like a LUT test polynomial: pre-rotated by half a box, the half box below
position 0 negated (X^N = -1), so that a blind rotation by the index, noise
included, lands inside the right box.  The interval index I is carried at
Delta_I = 2^(63 - log2 N_br) per interval with half an interval subtracted,
so that the rounding of the next blind rotation's modulus switch takes the
floor of Step 2.
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


# ---------------------------------------------------------------- encrypted lookup tables

def box_layout(values, N: int) -> list:
    """[N] Python ints: values[i] on box i (N / len(values) coefficients),
    pre-rotated by half a box, the half box below 0 holding -values[0]."""
    K = len(values)
    box = N // K
    h = box // 2
    return [values[(t + h) // box] if t < N - h else -values[0] for t in range(N)]


@dataclass
class EncodedLookup:
    p_hat: np.ndarray      # [N] int64
    q_hat: np.ndarray      # [N] uint64
    a_hat: np.ndarray      # [N_seg][N] int64
    b_hat: np.ndarray      # [N_seg][N] uint64
    N: int
    delta_x_log2: int      # x is carried as round(x 2^delta_x_log2)
    delta_r_log2: int      # values a x + b before the traces, per unit


def _pow2(v: int) -> bool:
    return v > 0 and v & (v - 1) == 0


def _i64(vals) -> np.ndarray:
    if any(abs(v) >= 1 << 63 for v in vals):
        raise ValueError("coefficient does not fit int64: lower the scales")
    return np.array(vals, dtype=np.int64)


def _u64(vals) -> np.ndarray:
    return np.array([v % (1 << 64) for v in vals], dtype=np.uint64)


def encode(lut: SegmentedLUT, N: int, delta_x_log2: int, delta_r_log2: int) -> EncodedLookup:
    """Integer polynomials of Steps 2 and 3 for ring size N:
    p, q with p_s = N_br/(tau_{s+1} - tau_s) Delta_I / Delta_x and
    q_s = -tau_s N_br/(tau_{s+1} - tau_s) Delta_I - Delta_I / 2;
    a_s, b_s with a_si Delta_r / Delta_x and b_si Delta_r per interval."""
    if not (_pow2(lut.n_seg) and _pow2(lut.n_br) and lut.n_seg <= N and lut.n_br <= N):
        raise ValueError("N_seg and N_br must be powers of two no larger than N")
    d_i = 1 << (63 - (lut.n_br.bit_length() - 1))
    w, q = index_polynomials(lut)
    sx = 2.0 ** -delta_x_log2
    p_vals = [round(float(w[s]) * d_i * sx) for s in range(lut.n_seg)]
    q_vals = [round(float(q[s]) * d_i) - d_i // 2 for s in range(lut.n_seg)]
    a_rows, b_rows = [], []
    for s in range(lut.n_seg):
        a_s, b_s = value_polynomials(lut, s)
        a_rows.append(_i64(box_layout([round(float(v) * 2.0 ** (delta_r_log2 - delta_x_log2)) for v in a_s], N)))
        b_rows.append(_u64(box_layout([round(float(v) * 2.0 ** delta_r_log2) for v in b_s], N)))
    return EncodedLookup(_i64(box_layout(p_vals, N)), _u64(box_layout(q_vals, N)), np.stack(a_rows),
                         np.stack(b_rows), N, delta_x_log2, delta_r_log2)


def encode_x(x: float, delta_x_log2: int) -> int:
    """Torus word carrying x in the constant coefficient of [[x]]."""
    return round(x * 2.0 ** delta_x_log2) % (1 << 64)


def segment_word(s: int, n_seg: int) -> int:
    """Torus word carrying the segment index S of [[S]] (Delta = 2^(63 - log2 N_seg))."""
    return (s << (63 - (n_seg.bit_length() - 1))) % (1 << 64)


def decode(phase0: int, enc: EncodedLookup) -> float:
    """f(x) from the constant coefficient of the lookup output's phase
    (N^2 a_SI x + b_SI in units of 2^-delta_r_log2: each trace multiplies by N)."""
    v = int(phase0) % (1 << 64)
    if v >= 1 << 63:
        v -= 1 << 64
    return v / (enc.N * enc.N * 2.0 ** enc.delta_r_log2)
