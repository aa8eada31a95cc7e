"""The largest-magnitude external product, with its closed form.

A GLWE whose every coefficient is C/2, C = sum_m (B/2) 2^(64 - m beta)
(m = 1..l), blind-rotated by one CMux with a~ = N: the CMux input
X^N ACC - ACC = -2 ACC = -C decomposes into digits that are all -B/2
(balanced digits of v are the plain base-B digits of v + C minus B/2, and
-C + C = 0).  Against key words of one sign and magnitude close to 2^63,
coefficient N-1 of the product sums (k+1) l N terms of one sign.

The product of the constant digit polynomial d (1 + X + ... + X^(N-1)) with a
key polynomial K in Z[X]/(X^N + 1) has coefficient t equal to
d (sum_{j<=t} K_j - sum_{j>t} K_j), so every output coefficient is known."""

import numpy as np

Q = 1 << 64


def case(p, sign, seed):
    """(bsk, lwe, glwe, C) for parameter set p: one LWE with a~_0 = N and
    every other a~_i = 0, b~ = 0; BSK words of sign `sign` (centred) and
    magnitude in (2^63 - 2^21, 2^63)."""
    B = 1 << p.pbs_base_log
    C = sum((B // 2) << (64 - m * p.pbs_base_log) for m in range(1, p.pbs_level + 1))
    g = np.random.default_rng(seed)
    small = g.integers(0, 1 << 20, size=p.bsk_shape(), dtype=np.uint64)
    if sign > 0:
        bsk = np.uint64(1 << 63) + np.uint64(1) + small         # centred -(2^63 - 1 - small)
    else:
        bsk = np.uint64((1 << 63) - 1) - small                  # centred +(2^63 - 1 - small)
    lwe = np.zeros((1, p.n + 1), np.uint64)
    lwe[0, 0] = np.uint64(1 << 63)
    glwe = np.full((1, p.k + 1, p.N), C // 2, np.uint64)
    return bsk, lwe, glwe, C


def centred(words):
    return [int(w) - Q if int(w) >= 1 << 63 else int(w) for w in np.asarray(words).reshape(-1)]


def expected(p, bsk, C):
    """The rotated GLWE, (k+1) x N Python ints mod 2^64, and the largest
    |sum| of one output coefficient before reduction."""
    B = 1 << p.pbs_base_log
    d = -(B // 2)
    out, peak = [], 0
    for c in range(p.k + 1):
        S = [0] * p.N
        for r in range(bsk.shape[1]):
            K = centred(bsk[0, r, c])
            total = sum(K)
            run = 0
            for t in range(p.N):
                run += K[t]
                S[t] += run - (total - run)
        peak = max(peak, max(abs(d * s) for s in S))
        out.append([(C // 2 + d * s) % Q for s in S])
    return out, peak
