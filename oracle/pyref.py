"""Independent pure-Python PBS on micro parameters — TEST INFRASTRUCTURE.

A second implementation of the same construction as ``tfhe_oracle.c``, written
separately with Python integers: polynomials are lists, products are full
linear convolutions folded by X^N = -1, rotations are list slices with sign
flips, gadget digits come from the balanced base-B expansion of the rounded
value.  It is only fast enough for micro parameters (N <= 64, n <= 16) and
serves to catch slips in the C oracle (overflow, off-by-one indexing).
"""

from __future__ import annotations

Q = 1 << 64
MASK = Q - 1


def negacyclic_mul(a, b):
    N = len(a)
    conv = [0] * (2 * N)
    for i, x in enumerate(a):
        if x:
            for j, y in enumerate(b):
                conv[i + j] += x * y
    return [(conv[t] - conv[t + N]) & MASK for t in range(N)]


def rotate(a, u):
    """X^u * a for any integer u (negacyclic)."""
    N = len(a)
    u %= 2 * N
    sign = 1
    if u >= N:
        u -= N
        sign = -1
    # X^u * a: coefficient t -> t + u, wrapping with a sign flip
    out = [0] * N
    for t in range(N):
        e = t + u
        if e < N:
            out[e] = (sign * a[t]) & MASK
        else:
            out[e - N] = (-sign * a[t]) & MASK
    return out


def gadget_digits(x, base_log, level):
    """Balanced base-2^base_log digits (most significant level first) of x
    rounded to its top base_log*level bits; the sum of digit_l * 2^(64 -
    l*base_log) equals the rounded value mod 2^64."""
    bits = base_log * level
    c = ((x + (1 << (63 - bits))) >> (64 - bits)) % (1 << bits) if bits < 64 else x
    B = 1 << base_log
    out = []
    for _ in range(level):              # least significant first
        d = c % B
        c //= B
        if d >= B // 2:
            d -= B
            c += 1
        out.append(d)
    return out[::-1]


def modswitch(x, two_n):
    return ((x * two_n + (Q >> 1)) // Q) % two_n


def pbs(params, s_lwe, bsk, ksk, lwe, lut):
    """params: dict n, k, N, base_log, level, ks_base_log, ks_level, msg_bits;
    bsk[i][row][c] lists of N ints; ksk[i][l] lists of n+1 ints."""
    n, k, N = params["n"], params["k"], params["N"]
    bl, lv = params["base_log"], params["level"]
    p = params["msg_bits"]
    box = N >> p
    h = box // 2
    v = [lut[(t + h) // box] if t < N - h else (-lut[0]) & MASK for t in range(N)]
    two_n = 2 * N
    b_t = modswitch(lwe[n], two_n)
    acc = [[0] * N for _ in range(k)] + [rotate(v, -b_t)]
    for i in range(n):
        a_t = modswitch(lwe[i], two_n)
        if a_t == 0:
            continue
        diff = [[(x - y) & MASK for x, y in zip(rotate(acc[j], a_t), acc[j])] for j in range(k + 1)]
        prod = [[0] * N for _ in range(k + 1)]
        for j in range(k + 1):
            digs = [gadget_digits(x, bl, lv) for x in diff[j]]
            for l in range(lv):
                dpoly = [d[l] & MASK for d in digs]
                row = bsk[i][j * lv + l]
                for c in range(k + 1):
                    pr = negacyclic_mul(dpoly, row[c])
                    prod[c] = [(x + y) & MASK for x, y in zip(prod[c], pr)]
        acc = [[(x + y) & MASK for x, y in zip(acc[c], prod[c])] for c in range(k + 1)]
    # extract constant coefficient
    big = []
    for j in range(k):
        A = acc[j]
        big += [A[0]] + [(-A[N - t]) & MASK for t in range(1, N)]
    big.append(acc[k][0])
    # key switch
    kbl, klv = params["ks_base_log"], params["ks_level"]
    out = [0] * n + [big[k * N]]
    for i in range(k * N):
        digs = gadget_digits(big[i], kbl, klv)
        for l in range(klv):
            row = ksk[i][l]
            out = [(o - digs[l] * r) & MASK for o, r in zip(out, row)]
    return out
