"""The CUDA path's explicit CRT, emulated on the CPU with exact integers.

The kernels reconstruct each external-product coefficient X (|X| <= 2^110
for every accepted parameter set) from four unreduced residues y_q < 8 p_q
that already carry the factor (M/p_q)^{-1}: X = sum_q y_q (M/p_q) - u M
(mod 2^64) with the quotient u taken from sum_q (y_q >> 2) / 2^26, not from
a reciprocal of each prime.  This checks that rule over random and extreme
X and representatives, with the primes read from the library's header."""

import os
import random
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "paper_2609_16915_gb300", "csrc", "internal.h")


def primes():
    text = open(HEADER).read()
    m = re.search(r"kPrimeList\[kPrimes\]\s*=\s*\{([^}]*)\}", text)
    return [int(v.strip().rstrip("u")) for v in m.group(1).split(",")]


def kernel_crt(X, ks, P):
    M = 1
    for p in P:
        M *= p
    ys = [((X % p) * pow((M // p) % p, -1, p)) % p + k * p for p, k in zip(P, ks)]
    assert all(y < 8 * p for y, p in zip(ys, P))
    ysum = sum(y >> 2 for y in ys)
    assert ysum < 2**31
    u = (ysum + (1 << 25)) >> 26
    s = sum(y * ((M // p) % 2**64) for y, p in zip(ys, P))
    return (s - u * (M % 2**64)) % 2**64


def test_primes_meet_the_stated_range():
    P = primes()
    assert len(P) == 4
    M = 1
    for p in P:
        assert 2**28 - 2**18 < p < 2**28
        assert (p - 1) % (1 << 14) == 0          # 2N-th roots of unity up to N = 8192
        assert all(p % d for d in range(2, int(p**0.5) + 1))      # prime (trial division)
        M *= p
    assert M > 2 * 2**110


@pytest.mark.parametrize("seed", range(4))
def test_quotient_from_shifted_sum_is_exact(seed):
    P = primes()
    B = 2**110
    rs = random.Random(seed)
    cases = [(X, ks) for X in (B, -B, 0, 1, -1) for ks in ([0] * 4, [7] * 4, [7, 0, 7, 0])]
    cases += [(rs.randint(-B, B), [rs.randint(0, 7) for _ in range(4)]) for _ in range(5000)]
    for X, ks in cases:
        assert kernel_crt(X, ks, P) == X % 2**64, (X, ks)


def test_a_wrong_quotient_rule_is_caught():
    """Rounding down instead of to nearest fails: the check can fail."""
    P = primes()
    M = 1
    for p in P:
        M *= p
    X = -(2**100)
    ys = [((X % p) * pow((M // p) % p, -1, p)) % p for p in P]
    u_floor = sum(y >> 2 for y in ys) >> 26
    s = sum(y * ((M // p) % 2**64) for y, p in zip(ys, P))
    assert (s - u_floor * (M % 2**64)) % 2**64 != X % 2**64
