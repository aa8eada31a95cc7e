"""The blind-rotation kernels' cross-CTA index arithmetic, modelled on the CPU.

Both kernels split a ciphertext's accumulator over the CTAs of a cluster and
exchange words through distributed shared memory by computed indices.  This
model follows the kernels' formulas (csrc/blind_rotate3.cu,
csrc/blind_rotate.cu) and checks them against the definitions they
implement:

* three-prime kernel: CTA o owns the first-pass slots [3o, min(3o+3, 8)) of
  every thread, i.e. coefficients tau + q T; phase 1 reads the source word
  of (X^a P)[j] = +-P[(j - a) mod 2N] from owner slot_owner(qs) at local
  slot qs - 3 os -- the gathered words must equal the negacyclic rotation;
* the residue exchanges of both kernels: the slot a producer writes a group
  to, and the slot its owner reads it from, must match for every producer,
  owner and thread, and cover each (producer, owner) pair once.
"""

import numpy as np
import pytest

S0 = (0, 3, 6, 8)  # first owned slot of the three owners, and the end


def slot_owner(q):
    """The kernel's two-bits-per-slot table: 0, 0, 0, 1, 1, 1, 2, 2."""
    return (0xA540 >> (2 * q)) & 3


def negacyclic_rotate(P, a):
    """(X^a P) mod X^N + 1 for integer coefficients."""
    N = len(P)
    out = [0] * N
    for i, v in enumerate(P):
        k = i + a
        sign = -1 if (k // N) % 2 else 1
        out[k % N] += sign * v
    return out


def test_slot_owner_table():
    assert [slot_owner(q) for q in range(8)] == [0, 0, 0, 1, 1, 1, 2, 2]
    for q in range(8):
        o = slot_owner(q)
        assert S0[o] <= q < S0[o + 1]


@pytest.mark.parametrize("L", [12, 13])
def test_three_prime_phase1_gather_is_the_negacyclic_rotation(L):
    """Every owned item of every owner reads, through the kernel's address
    formula, the word that makes (X^a P)[j] for several a~ (0 < a < 2N)."""
    N = 1 << L
    T = N // 8
    g = np.random.default_rng(L)
    P = [int(v) for v in g.integers(-(1 << 40), 1 << 40, N)]
    # each owner's shared array acc[c][h][tau] holds coefficient tau + (S0[o] + h) T
    acc = {o: {} for o in range(3)}
    for o in range(3):
        for h in range(S0[o + 1] - S0[o]):
            for tau in range(T):
                acc[o][(h, tau)] = P[tau + (S0[o] + h) * T]
    for at in (1, 7, N - 1, N, N + 3, 2 * N - 1, int(g.integers(1, 2 * N))):
        want = negacyclic_rotate(P, at)
        for o in range(3):
            for h in range(S0[o + 1] - S0[o]):
                for tau in range(T):
                    j = tau + (S0[o] + h) * T
                    e = (j + 2 * N - at) & (N - 1)
                    qs = e >> (L - 3)
                    os_ = slot_owner(qs)
                    hs = qs - 3 * os_
                    assert 0 <= hs < S0[os_ + 1] - S0[os_]
                    v = acc[os_][(hs, e & (T - 1))]
                    neg = ((j + 2 * N - at) & (2 * N - 1)) >= N
                    assert (-v if neg else v) == want[j], (at, o, h, tau)


def test_three_prime_residue_exchange_indices_match():
    """Producer r leaves owner o's group at index o < r ? o : o - 1 of its
    exchange buffer; owner o reads producer q's group at index
    o < q ? o : o - 1; the primes of an owner's remote slots 0 and 1 are
    (1, 2), (0, 2), (0, 1) for owners 0, 1, 2."""
    written = {}
    for r in range(3):
        for o in range(3):
            if o == r:
                continue
            oi = o if o < r else o - 1
            assert (r, oi) not in written
            written[(r, oi)] = o
    for o in range(3):
        q_r0 = 1 if o == 0 else 0
        q_r1 = 1 if o == 2 else 2
        assert sorted((q_r0, q_r1)) == sorted(set(range(3)) - {o})
        for q in (q_r0, q_r1):
            idx = o if o < q else o - 1
            assert written[(q, idx)] == o


def test_four_prime_residue_exchange_indices_match():
    """Prime-CTA r leaves owner o's group at [o][tau]; owner o reads group
    [o][tau] of every prime-CTA (its own included): one group per pair."""
    T = 32
    written = {}
    for r in range(4):
        for o in range(4):
            for tau in range(T):
                written[(r, o * T + tau)] = (o, tau)
    for o in range(4):
        for pq in range(4):
            for tau in range(T):
                assert written[(pq, o * T + tau)] == (o, tau)


@pytest.mark.parametrize("L", [12, 13])
def test_three_prime_digit_gather_places_every_slot(L):
    """Prime thread tau gathers, from owner o, the digits of slots
    [S0[o], S0[o+1]) as owner thread tau packed them (slots 0-1 in the 8-byte
    group, slot 2 in the 4-byte group of owners 0 and 1): the eight slots
    of its first pass, each exactly once."""
    filled = []
    for o in range(3):
        q = S0[o]
        filled += [q, q + 1]               # dig8: slots 0 and 1 of the owner
        if o < 2:
            filled.append(q + 2)           # dig4: slot 2
    assert sorted(filled) == list(range(8))
