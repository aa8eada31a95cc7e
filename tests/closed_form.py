"""Closed forms of PBS under noiseless keys, vectorised for full batches.

With a bootstrapping key whose GGSW rows have zero masks and zero noise,
every CMux step multiplies the accumulator by X^(a~_i s_i) exactly (the test
polynomial's words are multiples of Delta, which the gadget represents
exactly), so blind rotation returns the trivial GLWE (0, X^(-phi~) v) with
phi~ = b~ - sum_i a~_i s_i (mod 2N) the modulus-switched phase (Background,
"TFHE Scheme": the LUT is read off the rotated test polynomial's constant
term).  After extraction and a key switch with zero-mask, zero-noise rows the
output is (0, .., 0, F(m~)), m~ = round(phi~ / box) mod 2^(p+1) and F the LUT
extended negacyclically (F(m + 2^p) = -F(m)).

Only numpy here: no oracle code and no CUDA-library code.  The scalar form
of the same statement pins the oracle (tests/test_oracle.py); these
functions are checked against it on the CPU (tests/test_closed_form.py).
"""

from __future__ import annotations

import numpy as np

MASK64 = (1 << 64) - 1


def extended_lut(lut, msg_bits: int) -> np.ndarray:
    """F on [0, 2^(p+1)): lut[m] below 2^p, -lut[m - 2^p] (mod 2^64) above."""
    lut = np.asarray(lut, dtype=np.uint64)
    return np.concatenate([lut, (np.uint64(0) - lut).astype(np.uint64)])


def modswitch(words, N: int) -> np.ndarray:
    """round(x 2N / 2^64) mod 2N with ties rounded up, for uint64 words:
    (x + 2^(sh-1)) >> sh with sh = 64 - log2(2N); the sum wraps mod 2^64
    exactly when the rounded value is 2N, which is 0 mod 2N."""
    sh = 64 - (2 * N).bit_length() + 1
    x = np.asarray(words, dtype=np.uint64)
    return (((x + np.uint64(1 << (sh - 1))) >> np.uint64(sh)) & np.uint64(2 * N - 1)).astype(np.int64)


def switched_phase(params, lwe_key, lwe) -> np.ndarray:
    """phi~ = b~ - sum_i a~_i s_i mod 2N for every row of lwe [batch][n+1]."""
    ms = modswitch(lwe, params.N)
    s = np.asarray(lwe_key, dtype=np.int64)
    return (ms[:, params.n] - ms[:, :params.n] @ s) % (2 * params.N)


def noiseless_pbs_body(params, lwe_key, lwe, lut) -> np.ndarray:
    """Body word of PBS(lwe) under noiseless keys, one per row of lwe."""
    phi = switched_phase(params, lwe_key, np.atleast_2d(lwe))
    box = params.N >> params.msg_bits
    m = ((phi + box // 2) // box) % (1 << (params.msg_bits + 1))
    return extended_lut(lut, params.msg_bits)[m]


def noiseless_bsk(params, lwe_key) -> np.ndarray:
    """Raw bootstrapping key [n][(k+1)l][k+1][N] of GGSWs with zero masks
    and zero noise: row r = j l + (lev-1) of GGSW_i is zero except for
    s_i 2^(64 - lev beta) in the constant coefficient of component j (the
    GGSW definition with every GLWE encryption of zero taken noiseless)."""
    n, k, N, l, beta = params.n, params.k, params.N, params.pbs_level, params.pbs_base_log
    bsk = np.zeros((n, (k + 1) * l, k + 1, N), np.uint64)
    s = np.asarray(lwe_key, dtype=np.uint64)
    for j in range(k + 1):
        for lev in range(1, l + 1):
            bsk[:, j * l + lev - 1, j, 0] = s * np.uint64((1 << (64 - lev * beta)) & MASK64)
    return bsk


def noiseless_ksk(params, big_key) -> np.ndarray:
    """Raw key-switching key [kN][l_ks][n+1] of LWE rows with zero masks and
    zero noise: row [i][lev-1] = (0, .., 0, s'_i 2^(64 - lev beta_ks))."""
    kN, lk, n, bk = params.kN, params.ks_level, params.n, params.ks_base_log
    ksk = np.zeros((kN, lk, n + 1), np.uint64)
    sp = np.asarray(big_key, dtype=np.uint64).reshape(-1)
    for lev in range(1, lk + 1):
        ksk[:, lev - 1, n] = sp * np.uint64((1 << (64 - lev * bk)) & MASK64)
    return ksk
