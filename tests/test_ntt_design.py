"""The blind-rotation kernel's external-product arithmetic, emulated on the CPU.

A plain-Python model of what one cluster computes per CMux step and prime:
the register layout of the transforms (E = 8 values per thread, passes of
three stages with a shorter last pass, exchanges between passes), the twiddle
table W[m] = psi^bitrev(m) with Shoup companions, forward Cooley-Tukey
butterflies with the lazy correction schedule, the Montgomery
multiply-accumulate against keys that carry the CRT factor, inverse
Gentleman-Sande butterflies with the tracked correction rule, and the
explicit CRT with the shifted-sum quotient.  Every value is checked against
its documented bound (all below 2^32) and the result against the exact
negacyclic product mod 2^64 (numpy's wrapping uint64 convolution); a
separate pass propagates worst-case bounds through the same correction
schedule at every ring size, so the schedule is checked independently of
the data.  The rules mirror csrc/ntt.cuh, csrc/modarith.cuh and
csrc/blind_rotate.cu.

The three-prime kernel (csrc/blind_rotate3.cu) has its own model below:
primes just under 2^31, every transform value in [0, 2p), forward outputs
brought below p before the multiply-accumulate, row pairs accumulated in
[0, 2p), and the CRT quotient estimated against 2^31; exact up to the
largest magnitude the context accepts for it (0.45 of the primes' product)."""

import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
E, RAD = 8, 3
M32 = (1 << 32) - 1


def _prime_list(name):
    text = open(os.path.join(ROOT, "paper_2609_16915_gb300", "csrc", "internal.h")).read()
    m = re.search(name + r"\[\w+\]\s*=\s*\{([^}]*)\}", text)
    return [int(v.strip().rstrip("u")) for v in m.group(1).split(",")]


def primes():
    """The four 28-bit primes of the four-prime kernel."""
    return _prime_list("kPrimeList")


def primes31():
    """The three 31-bit primes of the three-prime kernel."""
    return _prime_list("kPrime31List")


def generator(p):
    f, n, d = [], p - 1, 2
    while d * d <= n:
        if n % d == 0:
            f.append(d)
            while n % d == 0:
                n //= d
        d += 1
    if n > 1:
        f.append(n)
    return next(g for g in range(2, p) if all(pow(g, (p - 1) // q, p) != 1 for q in f))


def bitrev(x, bits):
    return int(format(x, f"0{bits}b")[::-1], 2) if bits else 0


def twiddles(L, p):
    N = 1 << L
    psi = pow(generator(p), (p - 1) // (2 * N), p)
    assert pow(psi, N, p) == p - 1
    return [(w, (w << 32) // p) for w in (pow(psi, bitrev(m, L), p) for m in range(N))]


def passes(L):
    n = (L + RAD - 1) // RAD
    return [(RAD * i, RAD if i < n - 1 else L - RAD * (n - 1)) for i in range(n)]


def slot(L, S0, H, tau, e):
    """Position of register slot e of thread tau in the pass (S0, H)."""
    N = 1 << L
    SIG, SPAN, NB = N >> (S0 + H), N >> S0, E >> H
    b, q = e >> H, e & ((1 << H) - 1)
    beta = tau * NB + b
    return (beta // SIG) * SPAN + beta % SIG + q * SIG


def shoup(y, w, ws, p):
    assert 0 <= y <= M32
    q = (y * ws) >> 32
    r = (y * w - q * p) & M32
    assert r < 2 * p
    return r


def fwd_corrects(s):
    return s >= 7 and (s - 7) % 4 == 0


def inv_corrects(last, H, U, q):
    if U >= H - 1:
        return not last
    if (q >> (H - U - 2)) & 1:
        return False
    if U + 2 <= H - 1 and (q >> (H - U - 3)) & 1:
        return False
    return True


def exchange(L, xs, A, B):
    """Registers of pass A -> registers of pass B (through shared memory)."""
    T = (1 << L) // E
    buf = {}
    for tau in range(T):
        for e in range(E):
            buf[slot(L, A[0], A[1], tau, e)] = xs[tau][e]
    assert len(buf) == 1 << L                      # a permutation
    return [[buf[slot(L, B[0], B[1], tau, e)] for e in range(E)] for tau in range(T)]


def butterflies(L, S0, H, U):
    """(tau, register i0, register i1, group index) of every butterfly of
    stage S0 + U, in the kernel's order."""
    N, NB, HALF = 1 << L, E >> H, 1 << (H - 1 - U)
    SIG = N >> (S0 + H)
    for tau in range(N // E):
        for b in range(NB):
            g = (tau * NB + b) // SIG
            for q in range(1 << H):
                if not q & HALF:
                    yield tau, b * (1 << H) + q, b * (1 << H) + q + HALF, (g << U) + (q >> (H - U)), q


def forward(L, xs, tw, p):
    """Forward transform; inputs below 16p, outputs below 16p (bit-reversed)."""
    ps = passes(L)
    for pi, (S0, H) in enumerate(ps):
        for U in range(H):
            S = S0 + U
            for tau, i0, i1, G, _ in butterflies(L, S0, H, U):
                x = xs[tau]
                X, Y = x[i0], x[i1]
                assert X < 16 * p and Y < 16 * p
                if fwd_corrects(S):
                    X = min(X, (X - 8 * p) & M32)
                w, ws = tw[(1 << S) + G]
                t = shoup(Y, w, ws, p)
                x[i0], x[i1] = (X + t) & M32, (X - t + 2 * p) & M32
                assert x[i0] < 16 * p and x[i1] < 16 * p
        if pi + 1 < len(ps):
            xs = exchange(L, xs, ps[pi], ps[pi + 1])
    return xs


def inverse(L, xs, tw, p):
    """Inverse transform without N^-1; inputs below 8p, outputs below 8p."""
    ps = passes(L)
    for pi in range(len(ps) - 1, -1, -1):
        S0, H = ps[pi]
        for U in range(H - 1, -1, -1):
            S = S0 + U
            for tau, i0, i1, G, q in butterflies(L, S0, H, U):
                x = xs[tau]
                X, Y = x[i0], x[i1]
                assert X < 8 * p and Y < 8 * p
                s, d = X + Y, Y - X + 8 * p
                assert s < 16 * p and d < 16 * p
                if inv_corrects(pi == len(ps) - 1, H, U, q):
                    s = min(s, (s - 8 * p) & M32)
                assert s < 8 * p, "a skipped correction left a value at or above 8p"
                w, ws = tw[(2 << S) - 1 - G]
                x[i0], x[i1] = s, shoup(d, w, ws, p)
        if pi > 0:
            xs = exchange(L, xs, ps[pi], ps[pi - 1])
    return xs


def to_regs(L, poly):
    T = (1 << L) // E
    return [[poly[tau + e * T] for e in range(E)] for tau in range(T)]


def from_regs(L, xs):
    T = (1 << L) // E
    out = [0] * (1 << L)
    for tau in range(T):
        for e in range(E):
            out[tau + e * T] = xs[tau][e]
    return out


def redc(T, p, p_inv):
    assert T < p << 32
    m = (T * p_inv) & M32
    r = ((T >> 32) - ((m * p) >> 32) + p) & M32
    assert 0 < r < 2 * p
    return r


def external_product(L, digits, G, P):
    """sum_r digits[r] * G[r][c] for c = 0, 1 in Z_{2^64}[X]/(X^N + 1), the
    kernel's way (rows in pairs; keys transformed as at upload)."""
    N, R = 1 << L, len(digits)
    M = 1
    for p in P:
        M *= p
    ys = [[None] * len(P) for _ in range(2)]
    for qi, p in enumerate(P):
        tw, p_inv = twiddles(L, p), pow(p, -1, 1 << 32)
        crt_c = pow((M // p) % p, -1, p) * pow(N, -1, p) % p
        # keys: centred words mod p, forward transform, Montgomery form times the CRT factor
        Gh = []
        for r in range(R):
            per_c = []
            for c in range(2):
                centred = [(w - (1 << 64) if w >= 1 << 63 else w) % p for w in G[r][c]]
                fk = forward(L, to_regs(L, centred), tw, p)
                per_c.append([[(v % p) * (1 << 32) % p * crt_c % p for v in row] for row in fk])
            Gh.append(per_c)
        oh = None
        for r0 in range(0, R, 2):
            fx = [forward(L, to_regs(L, [(d + p) & M32 for d in digits[r0 + k]]), tw, p) for k in range(2)]
            acc = [[[0] * E for _ in range(N // E)] for _ in range(2)]
            for tau in range(N // E):
                for e in range(E):
                    x0 = min(fx[0][tau][e], (fx[0][tau][e] - 8 * p) & M32)
                    x1 = min(fx[1][tau][e], (fx[1][tau][e] - 8 * p) & M32)
                    for c in range(2):
                        rr = redc(x0 * Gh[r0][c][tau][e] + x1 * Gh[r0 + 1][c][tau][e], p, p_inv)
                        v = rr if oh is None else (oh[c][tau][e] + rr)
                        acc[c][tau][e] = v if oh is None else min(v, (v - 4 * p) & M32)
            oh = acc
        for c in range(2):
            y = from_regs(L, inverse(L, oh[c], tw, p))
            assert max(y) < 8 * p
            ys[c][qi] = y
    out = []
    for c in range(2):
        col = []
        for j in range(N):
            yq = [ys[c][qi][j] for qi in range(len(P))]
            s = sum(y * ((M // p) % 2**64) for y, p in zip(yq, P))
            u = (sum(y >> 2 for y in yq) + (1 << 25)) >> 26
            col.append((s - u * (M % 2**64)) % 2**64)
        out.append(col)
    return out


def negacyclic(a, b):
    """Exact product mod 2^64 in Z[X]/(X^N + 1) (uint64 arithmetic wraps)."""
    N = len(a)
    full = np.convolve(np.asarray(a, np.uint64), np.asarray(b, np.uint64))
    lo = full[:N].copy()
    lo[:N - 1] -= full[N:]
    return [int(v) for v in lo]


def expected(digits, G):
    out = []
    for c in range(2):
        tot = np.zeros(len(digits[0]), np.uint64)
        for r in range(len(digits)):
            tot += np.asarray(negacyclic([d % 2**64 for d in digits[r]], G[r][c]), np.uint64)
        out.append([int(v) for v in tot])
    return out


def test_convolution_reference_is_negacyclic():
    """X * X^(N-1) = X^N = -1, and a random product against a Python-int loop."""
    N = 8
    a = [0, 1] + [0] * (N - 2)
    b = [0] * (N - 1) + [1]
    assert negacyclic(a, b) == [2**64 - 1] + [0] * (N - 1)
    rs = np.random.default_rng(1)
    a = [int(v) for v in rs.integers(0, 2**64, N, dtype=np.uint64)]
    b = [int(v) for v in rs.integers(0, 2**64, N, dtype=np.uint64)]
    want = [0] * N
    for i in range(N):
        for j in range(N):
            k = (i + j) % N
            want[k] += a[i] * b[j] * (-1 if i + j >= N else 1)
    assert negacyclic(a, b) == [w % 2**64 for w in want]


@pytest.mark.parametrize("L,beta,R", [(8, 10, 4), (9, 16, 2), (10, 20, 2), (11, 23, 2)])
def test_emulated_external_product_is_exact(L, beta, R):
    N = 1 << L
    rs = np.random.default_rng(L)
    half = 1 << (beta - 1)
    digits = [[int(v) for v in rs.integers(-half, half, N)] for _ in range(R)]
    digits[0][0], digits[0][1] = -half, half - 1
    G = [[[int(v) for v in rs.integers(0, 2**64, N, dtype=np.uint64)] for _ in range(2)] for _ in range(R)]
    G[0][0][0], G[0][0][1] = 1 << 63, (1 << 63) - 1
    assert external_product(L, digits, G, primes()) == expected(digits, G)


def test_emulated_external_product_at_the_largest_magnitude():
    """Every digit -B/2 against every key word -2^63 (beta = 28, one level,
    N = 2048): coefficient N-1 is 2 N 2^27 2^63 = 2^102."""
    L, beta = 11, 28
    N = 1 << L
    digits = [[-(1 << (beta - 1))] * N for _ in range(2)]
    G = [[[1 << 63] * N for _ in range(2)] for _ in range(2)]
    assert external_product(L, digits, G, primes()) == expected(digits, G)


def worst_case_bounds(L):
    """Propagate the worst-case bound of every register (in units of p)
    through the kernel's forward transform, multiply-accumulate and inverse
    transform, with the same correction rules: a check of the schedule that
    does not depend on the data.  Returns the largest bound seen."""
    T, top = (1 << L) // E, 0
    ps = passes(L)
    b = [[2] * E for _ in range(T)]                  # digits + p: below 2p
    for pi, (S0, H) in enumerate(ps):
        for U in range(H):
            for tau, i0, i1, _, _ in butterflies(L, S0, H, U):
                bx = b[tau][i0]
                if fwd_corrects(S0 + U):
                    assert bx <= 16
                    bx = 8
                b[tau][i0] = b[tau][i1] = bx + 2     # X + t and X - t + 2p, t < 2p
                top = max(top, bx + 2)
                assert bx + 2 <= 16, f"forward stage {S0 + U} can exceed 16p"
        if pi + 1 < len(ps):
            b = exchange(L, b, ps[pi], ps[pi + 1])
    assert all(v <= 16 for row in b for v in row)
    # multiply-accumulate: inputs brought below 8p (16 p^2 < p 2^32), Montgomery
    # outputs below 2p, row pairs accumulated below 4p
    b = [[4] * E for _ in range(T)]
    for pi in range(len(ps) - 1, -1, -1):
        S0, H = ps[pi]
        for U in range(H - 1, -1, -1):
            for tau, i0, i1, _, q in butterflies(L, S0, H, U):
                bx, by = b[tau][i0], b[tau][i1]
                assert bx <= 8 and by <= 8
                s = bx + by
                assert s <= 16 and by + 8 <= 16
                if inv_corrects(pi == len(ps) - 1, H, U, q):
                    s = 8
                assert s <= 8, f"inverse stage {S0 + U} leaves a value that can reach {s}p"
                b[tau][i0], b[tau][i1] = s, 2
                top = max(top, s)
        if pi > 0:
            b = exchange(L, b, ps[pi], ps[pi - 1])
    return top


@pytest.mark.parametrize("L", range(8, 14))
def test_lazy_bounds_hold_in_the_worst_case(L):
    """Every ring size the kernels support: no value can reach 16p (and so
    2^32) in the forward transform, or 8p where the inverse skips a
    correction."""
    assert worst_case_bounds(L) <= 16
    assert 16 * max(primes()) < 2**32


# ---- the three-prime kernel: primes in (2^31 - 2^19, 2^31) ----

def cond(x, b):
    """min(x, x - b) on 32-bit words: x in [0, 2b) -> [0, b)."""
    return min(x, (x - b) & M32)


def forward31(L, xs, tw, p):
    """Forward transform with the P31 butterflies: inputs and outputs in [0, 2p)."""
    ps = passes(L)
    for pi, (S0, H) in enumerate(ps):
        for U in range(H):
            S = S0 + U
            for tau, i0, i1, G, _ in butterflies(L, S0, H, U):
                x = xs[tau]
                X, Y = x[i0], x[i1]
                assert X < 2 * p and Y < 2 * p
                w, ws = tw[(1 << S) + G]
                xr, t = cond(X, p), cond(shoup(Y, w, ws, p), p)
                assert xr < p and t < p
                x[i0], x[i1] = (xr + t) & M32, (xr - t + p) & M32
                assert x[i0] < 2 * p and x[i1] < 2 * p
        if pi + 1 < len(ps):
            xs = exchange(L, xs, ps[pi], ps[pi + 1])
    return xs


def inverse31(L, xs, tw, p):
    """Inverse transform (without N^-1) with the P31 butterflies: [0, 2p) in and out."""
    ps = passes(L)
    for pi in range(len(ps) - 1, -1, -1):
        S0, H = ps[pi]
        for U in range(H - 1, -1, -1):
            S = S0 + U
            for tau, i0, i1, G, _ in butterflies(L, S0, H, U):
                x = xs[tau]
                X, Y = x[i0], x[i1]
                assert X < 2 * p and Y < 2 * p
                xr, yr = cond(X, p), cond(Y, p)
                w, ws = tw[(2 << S) - 1 - G]
                x[i0], x[i1] = xr + yr, shoup((yr - xr + p) & M32, w, ws, p)
                assert x[i0] < 2 * p and x[i1] < 2 * p
        if pi > 0:
            xs = exchange(L, xs, ps[pi], ps[pi - 1])
    return xs


def crt_quotient31(ys):
    """round(sum y_q / p_q) estimated from the shifted sum against 2^31."""
    ysum = sum(y >> 3 for y in ys)
    assert ysum < 2**31
    return (ysum + (1 << 27)) >> 28


def external_product31(L, digits, G, P):
    """The three-prime kernel's external product (rows in pairs)."""
    N, R = 1 << L, len(digits)
    M = 1
    for p in P:
        M *= p
    ys = [[None] * len(P) for _ in range(2)]
    for qi, p in enumerate(P):
        assert 2**30 < p < 2**31
        tw, p_inv = twiddles(L, p), pow(p, -1, 1 << 32)
        crt_c = pow((M // p) % p, -1, p) * pow(N, -1, p) % p
        Gh = []
        for r in range(R):
            per_c = []
            for c in range(2):
                centred = [(w - (1 << 64) if w >= 1 << 63 else w) % p for w in G[r][c]]
                fk = forward31(L, to_regs(L, centred), tw, p)
                per_c.append([[cond(v, p) * (1 << 32) % p * crt_c % p for v in row] for row in fk])
            Gh.append(per_c)
        oh = None
        for r0 in range(0, R, 2):
            fx = [forward31(L, to_regs(L, [(d + p) & M32 for d in digits[r0 + k]]), tw, p) for k in range(2)]
            acc = [[[0] * E for _ in range(N // E)] for _ in range(2)]
            for tau in range(N // E):
                for e in range(E):
                    x0, x1 = cond(fx[0][tau][e], p), cond(fx[1][tau][e], p)
                    for c in range(2):
                        rr = redc(x0 * Gh[r0][c][tau][e] + x1 * Gh[r0 + 1][c][tau][e], p, p_inv)
                        acc[c][tau][e] = rr if oh is None else cond(oh[c][tau][e], p) + cond(rr, p)
                        assert acc[c][tau][e] < 2 * p
            oh = acc
        for c in range(2):
            y = from_regs(L, inverse31(L, oh[c], tw, p))
            assert max(y) < 2 * p
            ys[c][qi] = y
    out = []
    for c in range(2):
        col = []
        for j in range(N):
            yq = [ys[c][qi][j] for qi in range(len(P))]
            s = sum(y * ((M // p) % 2**64) for y, p in zip(yq, P))
            col.append((s - crt_quotient31(yq) * (M % 2**64)) % 2**64)
        out.append(col)
    return out


def test_three_prime_set():
    """Three primes c 2^14 + 1 in (2^31 - 2^19, 2^31): 2N | p - 1 up to
    N = 8192, 2p < 2^32, and a product above 2^92.999."""
    P = primes31()
    assert len(P) == 3 and len(set(P)) == 3
    for p in P:
        assert 2**31 - 2**19 < p < 2**31 and (p - 1) % 2**14 == 0
        assert p % 2 and all(p % d for d in range(3, int(p**0.5) + 1, 2))  # prime
    M = P[0] * P[1] * P[2]
    assert M > 2**92.999


def fits_three_primes(k, l, N, beta):
    """The context's rule: (k+1) l N 2^(beta-1) 2^63 <= 0.45 M3."""
    P = primes31()
    return (k + 1) * l * N * 2 ** (beta - 1) * 2**63 * 20 <= P[0] * P[1] * P[2] * 9


def test_three_prime_rule_and_quotient_margin():
    """The N = 4096 set (l = 2, beta = 15) and the N = 8192 one (l = 3,
    beta = 14) fit three primes, the N = 2048 set (l = 1, beta = 23) and
    N = 4096 with beta = 16 do not; and for every accepted bound the
    quotient estimate is off by less than 0.5 - 0.45."""
    assert fits_three_primes(1, 2, 4096, 15) and fits_three_primes(1, 3, 8192, 14)
    assert not fits_three_primes(1, 1, 2048, 23) and not fits_three_primes(1, 2, 4096, 16)
    P = primes31()
    # undershoot of y/2^31 against y/p for y < 2p, plus the shifted sum's truncation
    err = sum(2 * (2**31 - p) / 2**31 for p in P) + 3 * 8 / 2**31 + 2**-28
    assert err < 0.05


@pytest.mark.parametrize("L,beta,R", [(8, 15, 4), (9, 16, 2), (10, 14, 6), (12, 15, 4)])
def test_emulated_three_prime_external_product_is_exact(L, beta, R):
    N = 1 << L
    rs = np.random.default_rng(100 + L)
    half = 1 << (beta - 1)
    digits = [[int(v) for v in rs.integers(-half, half, N)] for _ in range(R)]
    digits[0][0], digits[0][1] = -half, half - 1
    G = [[[int(v) for v in rs.integers(0, 2**64, N, dtype=np.uint64)] for _ in range(2)] for _ in range(R)]
    G[0][0][0], G[0][0][1] = 1 << 63, (1 << 63) - 1
    assert external_product31(L, digits, G, primes31()) == expected(digits, G)


@pytest.mark.parametrize("L,beta,R", [(12, 15, 4), (12, 15, 6)])
def test_emulated_three_prime_external_product_at_the_largest_magnitude(L, beta, R):
    """Every digit -B/2 against every key word -2^63 at N = 4096: coefficient
    N-1 reaches R N 2^(beta-1) 2^63, 0.25 M3 with two levels (the N = 4096
    set) and 0.375 M3 with three (the largest bound a three-prime kernel
    accepts at this ring size)."""
    N = 1 << L
    P = primes31()
    assert R * N * 2 ** (beta - 1) * 2**63 <= 0.38 * P[0] * P[1] * P[2]
    digits = [[-(1 << (beta - 1))] * N for _ in range(R)]
    G = [[[1 << 63] * N for _ in range(2)] for _ in range(R)]
    assert external_product31(L, digits, G, P) == expected(digits, G)


# ---- the exchange buffer's padded layout ----

def xb_pad(kind, i):
    """The kernels' padding, 4 words after every 32 (kind 0); kind 1, 2 words
    after every 16, is the alternative the last test measures."""
    return i + ((i >> 5) << 2) if kind == 0 else i + ((i >> 4) << 1)


def pass_accesses(L, S0, H, kind):
    """Per warp and access instruction, the word addresses each thread
    touches (one for a scalar access; 4 or 2 consecutive words for the last
    pass's vector accesses), as the kernel computes them: a per-thread
    padded base plus a padded compile-time offset."""
    N, T = 1 << L, (1 << L) // E
    SIG, SPAN = N >> (S0 + H), N >> S0
    out = []
    for warp in range(max(1, T // 32)):
        ts = range(warp * 32, min(T, warp * 32 + 32))
        if SIG == 1:
            width = 4 if kind == 0 else 2
            for k in range(E // width):
                acc = []
                for t in ts:
                    base = xb_pad(kind, E * t)
                    assert xb_pad(kind, E * t + k * width) == base + k * width, "additive padding"
                    assert base % width == 0, "vector alignment"
                    acc.append([base + k * width + j for j in range(width)])
                out.append((width, acc))
        else:
            for q in range(E):
                acc = []
                for t in ts:
                    pos = (t // SIG) * SPAN + t % SIG
                    a = xb_pad(kind, pos) + xb_pad(kind, q * SIG)
                    assert a == xb_pad(kind, pos + q * SIG), "additive padding"
                    acc.append([a])
                out.append((1, acc))
    return out


def worst_bank_load(L, S0, H, kind):
    """Largest number of distinct words one bank serves in one warp access
    of the pass, over the ideal (1 per scalar access; 32 x width / 32 for
    vector accesses of `width` words)."""
    worst = 0
    for width, acc in pass_accesses(L, S0, H, kind):
        banks = {}
        for words in acc:
            for w in words:
                banks.setdefault(w % 32, set()).add(w)
        ideal = max(1, len(acc) * width // 32) if width > 1 else 1
        worst = max(worst, max(len(v) for v in banks.values()) / ideal)
    return worst


@pytest.mark.parametrize("L", range(8, 14))
def test_exchange_layout_in_bounds_bijective_and_nearly_conflict_free(L):
    """Every exchange of the transforms at every ring size: both passes'
    addresses are the same bijection of the N positions into N + N/8 words
    (additive in base and offset, vector accesses aligned), and every warp
    access is free of bank conflicts except in the one pass whose blocks
    have stride 2 (N = 1024 and 8192), which is two-way conflicted."""
    N = 1 << L
    ps = passes(L)
    for A, B in zip(ps, ps[1:]):
        kind = 0
        for S0, H in (A, B):
            SIG, SPAN = N >> (S0 + H), N >> S0
            seen = {}
            for t in range(N // E):
                for e in range(E):
                    pos = (t * E + e) if SIG == 1 else (t // SIG) * SPAN + t % SIG + e * SIG
                    seen[xb_pad(kind, pos)] = pos
            assert len(seen) == N and max(seen) < N + N // 8
            expect = 2 if (N >> (S0 + H)) == 2 else 1
            assert worst_bank_load(L, S0, H, kind) == expect, (L, (S0, H))


@pytest.mark.parametrize("L", [10, 13])
def test_alternative_padding_removes_the_stride_2_conflicts(L):
    """2 pad words after every 16 serves both passes of the two exchanges
    around the stride-2 pass without conflicts, but only with 8-byte vector
    accesses in the last pass (it breaks the 16-byte alignment).  Measured
    on the N = 8192 set it was 2.8 % slower (twice the last pass's
    accesses), so the kernels keep the single padding."""
    N = 1 << L
    ps = passes(L)
    k = [i for i, (S0, H) in enumerate(ps) if (N >> (S0 + H)) == 2][0]
    for S0, H in ps[k - 1:k + 2]:
        assert worst_bank_load(L, S0, H, 1) == 1
