"""The tensor-core key switch's exactness argument, emulated on the CPU.

The kernel cuts every 64-bit key word into `limbs` unsigned limbs, feeds the
signed key-switch digits and the limbs to bf16 tensor-core products with fp32
accumulation, and recombines the per-limb sums mod 2^64.  That is exact when
every digit and limb is an integer bf16 holds exactly (|v| <= 256) and every
partial sum stays below 2^24, which the library checks on the host:
2^(beta-1) (2^(64/limbs) - 1) K < 2^24 with K = kN l (8 limbs if that holds,
else 16, else the CUDA-core kernel).  Here the same digits (the closed form
the digit kernel uses), the same bf16 rounding (top half of the fp32 bits),
an fp32 matrix product and the same recombination are compared with the key
switch computed with exact integers, at the contraction lengths of the
benchmark's parameter sets, including the all-extreme case."""

import numpy as np
import pytest

import workload as W


def limbs_for(kN, level, base_log):
    """The host rule: limb count for exact fp32 sums, or 0."""
    if base_log > 8 or (kN * level) % 64:
        return 0
    K, dmax = kN * level, 1 << (base_log - 1)
    for limbs in (8, 16):
        if dmax * ((1 << (64 // limbs)) - 1) * K < 2**24:
            return limbs
    return 0


def digits_sequential(a, base_log, level):
    """Balanced digits the textbook way: round to the top beta l bits, then
    from the least significant level up, a digit >= B/2 becomes d - B with a
    carry.  Returns [level][...] with level 0 the most significant."""
    a = a.astype(object)
    bits = base_log * level
    B = 1 << base_log
    c = [(int(v) + (1 << (63 - bits))) >> (64 - bits) if bits < 64 else int(v) for v in a]
    out = [[0] * len(c) for _ in range(level)]
    for idx in range(len(c)):
        v = c[idx]
        for lev in range(level - 1, -1, -1):
            d = v & (B - 1)
            v >>= base_log
            if d >= B // 2:
                d -= B
                v += 1
            out[lev][idx] = d
    return np.array(out, dtype=np.int64)


def digits_closed_form(a, base_log, level):
    """The digit kernel's rule: plain base-B digits of v + sum_m (B/2) B^m,
    minus B/2."""
    bits = base_log * level
    B = 1 << base_log
    C = sum((B >> 1) << (m * base_log) for m in range(level))
    out = np.zeros((level, len(a)), np.int64)
    for idx, x in enumerate(a):
        v = int(x)
        v = v if bits >= 64 else (v + (1 << (63 - bits))) >> (64 - bits)
        v = (v + C) & ((1 << bits) - 1) if bits < 64 else (v + C) % 2**64
        for lev in range(level):
            sh = base_log * (level - 1 - lev)
            out[lev, idx] = ((v >> sh) & (B - 1)) - (B >> 1)
    return out


def bf16(x):
    """Round-toward-zero to bf16 the way the tile kernels do (top half of
    the fp32 bits), returned as float32."""
    u = np.asarray(x, np.float32).view(np.uint32) & np.uint32(0xFFFF0000)
    return u.view(np.float32)


def keyswitch_tc(big, ksk, n, base_log, level, limbs):
    """[batch][kN+1] -> [batch][n+1] the tensor-core kernel's way."""
    batch, kN = big.shape[0], big.shape[1] - 1
    lbits = 64 // limbs
    d = np.stack([digits_closed_form(big[b, :kN], base_log, level) for b in range(batch)])  # [b][lev][i]
    A = d.transpose(0, 1, 2).reshape(batch, level * kN)             # r = lev kN + i (level-major)
    Af = bf16(A.astype(np.float32))
    assert np.array_equal(Af.astype(np.int64), A)                     # digits exact in bf16
    K = ksk.transpose(1, 0, 2).reshape(level * kN, n + 1)             # KSK[i][lev][j] -> row lev kN + i
    s = np.zeros((batch, n + 1), np.uint64)
    for t in range(limbs):
        Lt = ((K >> np.uint64(lbits * t)) & np.uint64((1 << lbits) - 1)).astype(np.int64)
        Lf = bf16(Lt.astype(np.float32))
        assert np.array_equal(Lf.astype(np.int64), Lt)                # limbs exact in bf16
        Ct = Af @ Lf                                                   # fp32 accumulation
        ci = np.rint(Ct).astype(np.int64)
        s += ci.astype(np.uint64) << np.uint64(lbits * t)
    out = np.zeros((batch, n + 1), np.uint64)
    out[:, n] = big[:, kN]
    return out - s


def keyswitch_exact(big, ksk, n, base_log, level):
    batch, kN = big.shape[0], big.shape[1] - 1
    out = np.zeros((batch, n + 1), np.uint64)
    out[:, n] = big[:, kN]
    for b in range(batch):
        d = digits_sequential(big[b, :kN], base_log, level)           # [lev][i]
        acc = np.zeros(n + 1, np.uint64)
        for lev in range(level):
            acc += d[lev].astype(np.uint64) @ ksk[:, lev, :]            # wraps mod 2^64
        out[b] -= acc
    return out


# (kN, l_ks, beta_ks) of the parameter sets and the limb count the rule gives
SETS = {name: (W.CONFIGS[name].k * W.CONFIGS[name].N, W.CONFIGS[name].ks_level, W.CONFIGS[name].ks_base_log)
        for name in ("tiny", "standard", "gpt2_mlp", "llama_silu")}


def test_limb_rule_for_the_parameter_sets():
    assert {k: limbs_for(*v) for k, v in SETS.items()} == {"tiny": 8, "standard": 8, "gpt2_mlp": 16, "llama_silu": 16}
    assert limbs_for(2048, 5, 9) == 0                  # beta > 8: left to the CUDA-core kernel
    assert limbs_for(2056, 1, 3) == 0                  # K not a multiple of the 64-wide MMA step
    assert limbs_for(8192, 8, 8) == 0                  # no limb count keeps the sums below 2^24


@pytest.mark.parametrize("base_log,level", [(3, 5), (4, 6), (8, 8), (16, 4), (1, 64)])
def test_closed_form_digits_equal_the_carry_rule(base_log, level):
    rs = np.random.default_rng(base_log * 100 + level)
    a = rs.integers(0, 2**64, 4000, dtype=np.uint64)
    bits = base_log * level
    edge = [0, 2**64 - 1, 2**63, 2**63 - 1]
    if bits < 64:
        half = 1 << (63 - bits)
        edge += [half, half - 1, 2**64 - half, (3 * half) % 2**64]
    a = np.concatenate([a, np.array(edge, np.uint64)])
    assert np.array_equal(digits_closed_form(a, base_log, level), digits_sequential(a, base_log, level))


def _words_with_plain_digit(one, base_log, level):
    """A torus word whose every plain digit of v + C equals `one`."""
    B, bits = 1 << base_log, base_log * level
    v = sum(((one - B // 2) % B) * B**m for m in range(level)) % 2**bits
    return np.uint64((v << (64 - bits)) % 2**64)


@pytest.mark.parametrize("name", sorted(SETS))
def test_tensor_core_keyswitch_is_exact(name):
    kN, level, base_log = SETS[name]
    limbs, n = limbs_for(kN, level, base_log), 16
    rs = np.random.default_rng(len(name))
    big = rs.integers(0, 2**64, (3, kN + 1), dtype=np.uint64)
    ksk = rs.integers(0, 2**64, (kN, level, n + 1), dtype=np.uint64)
    assert np.array_equal(keyswitch_tc(big, ksk, n, base_log, level, limbs), keyswitch_exact(big, ksk, n, base_log, level))
    # the largest partial sums the rule allows: every digit -B/2 (or 1 - B/2,
    # odd) against every limb at its maximum
    for one in (0, 1):
        big = np.full((2, kN + 1), _words_with_plain_digit(one, base_log, level), np.uint64)
        ksk = np.full((kN, level, n + 1), 2**64 - 1, np.uint64)
        got = keyswitch_tc(big, ksk, n, base_log, level, limbs)
        assert np.array_equal(got, keyswitch_exact(big, ksk, n, base_log, level))


def test_fewer_limbs_than_the_rule_asks_are_not_exact():
    """The bound matters: at the gpt2_mlp contraction length, 8-bit limbs
    against odd digits push the fp32 sums past 2^24 and the words differ."""
    kN, level, base_log = SETS["gpt2_mlp"]
    assert limbs_for(kN, level, base_log) == 16
    n = 4
    big = np.full((1, kN + 1), _words_with_plain_digit(1, base_log, level), np.uint64)
    ksk = np.full((kN, level, n + 1), 2**64 - 1, np.uint64)
    assert not np.array_equal(keyswitch_tc(big, ksk, n, base_log, level, 8), keyswitch_exact(big, ksk, n, base_log, level))
