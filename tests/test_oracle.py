"""Pins of the CPU oracle against facts that do not come from the oracle:
brute-force ring products, exhaustive toy-width gadget/modulus-switch checks,
the paper's worked rotation example, closed forms under noiseless keys, the
decryption invariant of PBS and noise bounds of the key switch."""

import json
import os
import random

import numpy as np
import pytest

import oracle as O
import workload as W
from oracle import pyref

GOLD = os.path.join(os.path.dirname(__file__), "golden")
Q = 1 << 64
M64 = Q - 1


def rnd_u64(rs, n):
    return np.array([rs.getrandbits(64) for _ in range(n)], dtype=np.uint64)


# ------------------------------------------------------------------ ring

@pytest.mark.parametrize("N", [1, 2, 4, 8, 16, 64])
def test_poly_mul_matches_integer_convolution(N):
    """Product in Z_{2^64}[X]/(X^N+1): exact integer convolution, then fold
    with X^N = -1, then reduce mod 2^64 (ring definition, Background,
    Notation)."""
    rs = random.Random(N)
    for _ in range(5):
        a = [rs.getrandbits(64) for _ in range(N)]
        b = [rs.getrandbits(64) for _ in range(N)]
        full = [0] * (2 * N - 1)
        for i in range(N):
            for j in range(N):
                full[i + j] += a[i] * b[j]
        want = [(full[t] - (full[t + N] if t + N < 2 * N - 1 else 0)) % Q for t in range(N)]
        got = O.poly_mul(np.array(a, np.uint64), np.array(b, np.uint64))
        assert [int(x) for x in got] == want


def test_ring_identities():
    rs = random.Random(7)
    N = 32
    a, b, c = rnd_u64(rs, N), rnd_u64(rs, N), rnd_u64(rs, N)
    # commutativity and distributivity
    assert np.array_equal(O.poly_mul(a, b), O.poly_mul(b, a))
    assert np.array_equal(O.poly_mul(a, b + c), O.poly_mul(a, b) + O.poly_mul(a, c))
    # X^N = -1 and X^{2N} = 1
    assert np.array_equal(O.poly_monomial(a, N), (np.uint64(0) - a))
    assert np.array_equal(O.poly_monomial(a, 0), a)
    for u in [1, 5, N - 1, N + 3, 2 * N - 1]:
        mono = np.zeros(N, np.uint64)
        if u < N:
            mono[u] = 1
        else:
            mono[u - N] = np.uint64(M64)        # X^u = -X^(u-N)
        assert np.array_equal(O.poly_monomial(a, u), O.poly_mul(a, mono)), u
        # X^u X^v = X^(u+v)
        v = (3 * u + 1) % (2 * N)
        assert np.array_equal(O.poly_monomial(O.poly_monomial(a, u), v), O.poly_monomial(a, (u + v) % (2 * N)))


def test_paper_rotation_example():
    """Left rotation by m puts f(m) in the constant coefficient."""
    g = json.load(open(os.path.join(GOLD, "paper_rotation_example.json")))
    lut = np.array(g["lut"], np.uint64)
    N = len(lut)
    rotated = O.poly_monomial(lut, 2 * N - g["m"])          # X^{-m}
    assert int(rotated[0]) == g["constant_term"]
    # the same with the box layout of the test polynomial (box = 2)
    v = O.test_poly(lut, 2, 2 * N)
    assert int(O.poly_monomial(v, 4 * N - g["m"] * 2)[0]) == g["constant_term"]


def test_paper_staircase_example():
    g = json.load(open(os.path.join(GOLD, "paper_staircase_example.json")))
    mids = W.bin_midpoints(g["lo"], g["hi"], g["entries"])
    d = g["printed_decimals"]
    assert round(mids[0], d) == pytest.approx(g["first_midpoint"], abs=10 ** -d)
    assert round(1.0 / mids[0], d) == pytest.approx(g["first_entry"], abs=10 ** -d)
    assert g["lo"] + (g["hi"] - g["lo"]) / g["entries"] == pytest.approx(g["first_interval_end"])
    assert W.bin_index(g["query"], g["lo"], g["hi"], g["entries"]) == g["index"]
    assert W.bin_index(g["query"], *g["segment"], g["entries"]) == g["segment_index"]


# ------------------------------------------------------------------ gadget / modswitch

TOY = 16


@pytest.mark.parametrize("base_log,level", [(2, 8), (3, 5), (4, 4), (5, 3), (8, 2), (16, 1), (4, 3), (1, 7)])
def test_decompose_exhaustive_16bit_torus(base_log, level):
    """Every 16-bit torus value x*2^48: digits lie in [-B/2, B/2) and
    recompose to x rounded (half up) to its top base_log*level bits."""
    bits = base_log * level
    B = 1 << base_log
    for x16 in range(1 << TOY):
        x = x16 << (64 - TOY)
        d = O.decompose(x, base_log, level)
        assert all(-B // 2 <= v < B // 2 for v in d)
        rec = sum(v * (1 << (64 - (l + 1) * base_log)) for l, v in enumerate(d)) % Q
        # nearest multiple of 2^(64-bits), ties up
        step = 1 << (64 - bits)
        want = ((x + step // 2) // step * step) % Q
        assert rec == want


def test_decompose_random_64bit_all_configs():
    rs = random.Random(3)
    pairs = set()
    for p in W.CONFIGS.values():
        pairs.add((p.pbs_base_log, p.pbs_level))
        pairs.add((p.ks_base_log, p.ks_level))
    for base_log, level in sorted(pairs):
        B, bits = 1 << base_log, base_log * level
        step = 1 << (64 - bits)
        for _ in range(2000):
            x = rs.getrandbits(64)
            d = O.decompose(x, base_log, level)
            assert all(-B // 2 <= v < B // 2 for v in d)
            rec = sum(v * (1 << (64 - (l + 1) * base_log)) for l, v in enumerate(d)) % Q
            assert rec == ((x + step // 2) // step * step) % Q
            assert d == pyref.gadget_digits(x, base_log, level)


@pytest.mark.parametrize("log2_2N", [1, 2, 5, 9, 12])
def test_modswitch_exhaustive_16bit_torus(log2_2N):
    two_n = 1 << log2_2N
    for x16 in range(1 << TOY):
        x = x16 << (64 - TOY)
        # round(x * 2N / 2^64), ties up, mod 2N -- exact rational arithmetic
        want = ((2 * x * two_n + Q) // (2 * Q)) % two_n
        assert O.modswitch(x, log2_2N) == want


# ------------------------------------------------------------------ extraction

@pytest.mark.parametrize("k,N", [(1, 16), (2, 8), (1, 256)])
def test_sample_extract_phase_is_constant_coefficient(k, N):
    """phase(extract(C)) equals coefficient 0 of phase(C), exactly."""
    rs = random.Random(k * 100 + N)
    S = np.array([[rs.getrandbits(1) for _ in range(N)] for _ in range(k)], np.uint64)
    for _ in range(10):
        ct = rnd_u64(rs, (k + 1) * N).reshape(k + 1, N)
        lwe = O.sample_extract(ct)
        assert int(O.lwe_phase(S.reshape(-1), lwe)[0]) == int(O.glwe_phase(S, ct)[0])


# ------------------------------------------------------------------ external product / CMux

def _round_top(x, bits):
    step = 1 << (64 - bits)
    return ((x + step // 2) // step * step) % Q


def test_external_product_noiseless_closed_form():
    """With a GGSW of mu that has zero masks and zero noise, the external
    product equals mu * (each coefficient rounded to its top base_log*level
    bits), component by component."""
    rs = random.Random(11)
    k, N, bl, lv = 1, 16, 6, 3
    S = np.array([[rs.getrandbits(1) for _ in range(N)] for _ in range(k)], np.uint64)
    zero_mask = np.zeros(((k + 1) * lv, k, N), np.uint64)
    zero_noise = np.zeros(((k + 1) * lv, N), np.uint64)
    for mu in [0, 1, 3]:
        ggsw = O.ggsw_encrypt(S, mu, bl, lv, zero_mask, zero_noise)
        C = rnd_u64(rs, (k + 1) * N).reshape(k + 1, N)
        got = O.external_product(ggsw, C, bl, lv)
        want = np.array([[(mu * _round_top(int(x), bl * lv)) % Q for x in row] for row in C], np.uint64)
        assert np.array_equal(got, want)


def test_external_product_decrypts_to_mu_times_message():
    """GGSW(mu) (x) GLWE(M): phase close to mu*M, error within the bound
    sum_{j,l} |D_jl| * |e_row| + mu * (k+1 rounding errors)."""
    rs = random.Random(12)
    k, N, bl, lv = 1, 32, 8, 3
    g = np.random.default_rng(5)
    S = np.array([[rs.getrandbits(1) for _ in range(N)] for _ in range(k)], np.uint64)
    sigma = 2 ** 20
    for mu in [0, 1]:
        mask = rnd_u64(rs, (k + 1) * lv * k * N).reshape((k + 1) * lv, k, N)
        noise = np.rint(g.standard_normal(((k + 1) * lv, N)) * sigma).astype(np.int64).view(np.uint64)
        ggsw = O.ggsw_encrypt(S, mu, bl, lv, mask, noise)
        M = (np.array([rs.getrandbits(4) for _ in range(N)], np.uint64) << np.uint64(60))
        ct = O.glwe_encrypt(S, M, rnd_u64(rs, k * N).reshape(k, N), np.zeros(N, np.uint64))
        out = O.external_product(ggsw, ct, bl, lv)
        ph = O.glwe_phase(S, out).astype(object)
        want = (M.astype(object) * mu) % Q
        err = [((int(a) - int(b) + Q // 2) % Q) - Q // 2 for a, b in zip(ph, want)]
        max_e = int(np.max(np.abs(noise.view(np.int64))))
        bound = (k + 1) * lv * N * (1 << (bl - 1)) * max_e + (1 + k * N) * (1 << (63 - bl * lv))
        assert max(abs(e) for e in err) <= bound


# ------------------------------------------------------------------ PBS

def _extended_lut(lut, p):
    """Negacyclic extension F(m), m in [0, 2^(p+1)): lut[m], then -lut[m-2^p]."""
    return [int(x) for x in lut] + [(-int(x)) % Q for x in lut]


def _closed_form_pbs(params, s, lwe, lut):
    """PBS with noiseless keys returns the trivial LWE (0, .., 0, F(m~)) where
    phi~ = b~ - sum a~_i s_i (mod 2N) is the modulus-switched phase and
    m~ = round(phi~ / box) mod 2^(p+1), box = N / 2^p."""
    N, p = params.N, params.msg_bits
    two_n = 2 * N
    ms = [((2 * int(x) * two_n + Q) // (2 * Q)) % two_n for x in lwe]
    phi = (ms[-1] - sum(ms[i] * int(s[i]) for i in range(params.n))) % two_n
    box = N >> p
    m = ((phi + box // 2) // box) % (1 << (p + 1))
    return _extended_lut(lut, p)[m]


@pytest.mark.parametrize("cfg", ["tiny"])
def test_pbs_noiseless_keys_closed_form(cfg):
    p = W.CONFIGS[cfg]
    keys = O.Keys(p, W.key_draws(p, trivial=True))
    lut = W.lut_torus(p, codes=[(3 * m + 1) % (1 << p.msg_bits) for m in range(1 << p.msg_bits)])
    lwe = W.uniform_ciphertexts(p, 48)          # any words: not encryptions
    out = O.pbs_batch(p, keys.bsk, keys.ksk, lwe, lut)
    for b in range(lwe.shape[0]):
        assert not out[b, :p.n].any()
        assert int(out[b, p.n]) == _closed_form_pbs(p, keys.lwe_key, lwe[b], lut)


def test_pbs_decrypts_to_lut_tiny():
    """decrypt(PBS(Enc(m))) == LUT(m) for every message (Background, TFHE
    Scheme: TFHE-LUT_f([[m]]) = [[f(m)]]); tiny parameters have a noise
    margin of many standard deviations, so no failures are expected."""
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p))
    codes = np.tile(np.arange(1 << p.msg_bits), 64)
    cts = keys.encrypt(W.cipher_draws(p, codes.size, codes=codes, sub=1))
    lut = W.lut_torus(p)
    out = O.pbs_batch(p, keys.bsk, keys.ksk, cts, lut)
    assert np.array_equal(keys.decrypt(out), W.lut_codes(p)[codes])
    big = O.blind_rotate_extract_batch(p, keys.bsk, cts[:16], lut)
    assert np.array_equal(keys.decrypt_big(big), W.lut_codes(p)[codes[:16]])


def test_pbs_matches_independent_python_micro():
    """Bit-exact agreement with the separately written pure-Python PBS."""
    from workload import Params
    p = Params("micro", n=6, k=1, N=16, pbs_base_log=7, pbs_level=2, ks_base_log=3, ks_level=3,
               msg_bits=2, lwe_sigma_log2=30, glwe_sigma_log2=30, lut=("square_mod",),
               msg=("uniform",), batch=4, seed=42)
    keys = O.Keys(p, W.key_draws(p))
    lut = W.lut_torus(p, codes=[1, 3, 0, 2])
    lwe = W.uniform_ciphertexts(p, 6)
    got = O.pbs_batch(p, keys.bsk, keys.ksk, lwe, lut)
    prm = dict(n=p.n, k=p.k, N=p.N, base_log=p.pbs_base_log, level=p.pbs_level,
               ks_base_log=p.ks_base_log, ks_level=p.ks_level, msg_bits=p.msg_bits)
    bsk = [[[list(map(int, keys.bsk[i, r, c])) for c in range(p.k + 1)] for r in range(keys.bsk.shape[1])]
           for i in range(p.n)]
    ksk = [[list(map(int, keys.ksk[i, l])) for l in range(p.ks_level)] for i in range(p.kN)]
    for b in range(lwe.shape[0]):
        want = pyref.pbs(prm, None, bsk, ksk, list(map(int, lwe[b])), list(map(int, lut)))
        assert [int(x) for x in got[b]] == want


# ------------------------------------------------------------------ key switch

def test_keyswitch_trivial_shift_is_exact():
    """KS(c + (0,..,0,delta)) = KS(c) + (0,..,0,delta): the body never enters
    the decomposition."""
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p))
    rs = random.Random(4)
    big = rnd_u64(rs, 4 * (p.kN + 1)).reshape(4, p.kN + 1)
    delta = np.uint64(rs.getrandbits(64))
    a = O.keyswitch_batch(p, keys.ksk, big)
    big2 = big.copy()
    big2[:, -1] += delta
    b = O.keyswitch_batch(p, keys.ksk, big2)
    assert np.array_equal(b[:, :-1], a[:, :-1])
    assert np.array_equal(b[:, -1], a[:, -1] + delta)


def test_keyswitch_preserves_phase_within_bound():
    """|phase_s(KS(c)) - phase_s'(c)| <= sum_{i,l} |d_il| |e_il| + kN * 2^(63 -
    ks_base_log*ks_level) (decomposition rounding), with the actual noises."""
    p = W.CONFIGS["tiny"]
    draws = W.key_draws(p)
    keys = O.Keys(p, draws)
    rs = random.Random(9)
    big = rnd_u64(rs, 6 * (p.kN + 1)).reshape(6, p.kN + 1)
    out = O.keyswitch_batch(p, keys.ksk, big)
    e = np.abs(draws.ksk_noise.view(np.int64)).astype(object)
    half_b = 1 << (p.ks_base_log - 1)
    bound = int(sum(e.reshape(-1))) * half_b + p.kN * (1 << (63 - p.ks_base_log * p.ks_level))
    for b in range(big.shape[0]):
        ph_out = int(O.lwe_phase(keys.lwe_key, out[b])[0])
        ph_in = int(O.lwe_phase(keys.big_key, big[b])[0])
        diff = ((ph_out - ph_in + Q // 2) % Q) - Q // 2
        assert abs(diff) <= bound


def test_keyswitch_noiseless_key_closed_form():
    """With zero-mask, zero-noise KSK rows (0,..,0, s'_i 2^(64-l beta)), the
    output is (0,..,0, b' - sum_i s'_i round(a'_i))."""
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p, trivial=True))
    rs = random.Random(10)
    big = rnd_u64(rs, 3 * (p.kN + 1)).reshape(3, p.kN + 1)
    out = O.keyswitch_batch(p, keys.ksk, big)
    bits = p.ks_base_log * p.ks_level
    for b in range(3):
        assert not out[b, :-1].any()
        want = (int(big[b, -1]) - sum(int(keys.big_key[i]) * _round_top(int(big[b, i]), bits)
                                      for i in range(p.kN))) % Q
        assert int(out[b, -1]) == want


# ------------------------------------------------------------------ blind rotation of an encrypted test polynomial

def test_glwe_blind_rotation_of_trivial_glwe_is_the_lut_path():
    """Rotating the trivial GLWE (0, v) must reproduce the public-LUT blind
    rotation word for word."""
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p))
    lut = W.lut_torus(p)
    v = O.test_poly(lut, p.msg_bits, p.N)
    lwe = W.uniform_ciphertexts(p, 3, sub=11)
    glwe = np.zeros((3, p.k + 1, p.N), np.uint64)
    glwe[:, p.k] = v
    got = O.blind_rotate_glwe_batch(p, keys.bsk, lwe, glwe)
    for b in range(3):
        assert np.array_equal(got[b], O.blind_rotate(p, keys.bsk, lwe[b], lut))


def test_glwe_blind_rotation_noiseless_closed_form():
    """With noiseless keys and input words that are multiples of 2^(64 -
    base_log*level) (so the gadget rounding is exact), the output is exactly
    X^{-phi~} times the input GLWE, phi~ the modulus-switched phase."""
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p, trivial=True))
    rs = np.random.default_rng(8)
    shift = np.uint64(64 - p.pbs_base_log * p.pbs_level)
    glwe = (rs.integers(0, 2**63, size=(4, p.k + 1, p.N), dtype=np.uint64) << shift).astype(np.uint64)
    lwe = W.uniform_ciphertexts(p, 4, sub=12)
    got = O.blind_rotate_glwe_batch(p, keys.bsk, lwe, glwe)
    two_n = 2 * p.N
    for b in range(4):
        ms = [((2 * int(x) * two_n + Q) // (2 * Q)) % two_n for x in lwe[b]]
        phi = (ms[-1] - sum(ms[i] * int(keys.lwe_key[i]) for i in range(p.n))) % two_n
        for c in range(p.k + 1):
            assert np.array_equal(got[b, c], O.poly_monomial(glwe[b, c], (two_n - phi) % two_n))


def test_glwe_blind_rotation_decrypts_to_rotated_table():
    """Real keys, an encrypted test polynomial: the GLWE phase of the output
    holds the table rotated left by the encrypted message (its constant
    coefficient decodes to LUT(m))."""
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p))
    codes = np.arange(8)
    cts = keys.encrypt(W.cipher_draws(p, 8, codes=codes, sub=13))
    lut = W.lut_torus(p)
    v = O.test_poly(lut, p.msg_bits, p.N)
    g = W.rng(p.seed, "sample", 13)
    glwe = np.stack([O.glwe_encrypt(keys.glwe_key, v, W.uniform_u64((p.k, p.N), g),
                                    W.gaussian_u64((p.N,), p.glwe_sigma_log2, g)) for _ in range(8)])
    out = O.blind_rotate_glwe_batch(p, keys.bsk, cts, glwe)
    sh = 63 - p.msg_bits
    for b in range(8):
        ph = int(O.glwe_phase(keys.glwe_key, out[b])[0])
        assert ((ph + (1 << (sh - 1))) >> sh) % (1 << (p.msg_bits + 1)) == W.lut_codes(p)[codes[b]]


# ------------------------------------------------------------------ RLWE trace

@pytest.mark.parametrize("N", [8, 64])
def test_automorphism_is_a_ring_homomorphism(N):
    rs = random.Random(N + 1)
    a, b = rnd_u64(rs, N), rnd_u64(rs, N)
    for k in [1, 3, 5, N + 1, 2 * N - 1]:
        assert np.array_equal(O.automorphism(O.poly_mul(a, b), k), O.poly_mul(O.automorphism(a, k), O.automorphism(b, k)))
        for k2 in [3, N - 1]:
            assert np.array_equal(O.automorphism(O.automorphism(a, k), k2), O.automorphism(a, (k * k2) % (2 * N)))
    assert np.array_equal(O.automorphism(a, 1), a)
    # X -> X^(N+1) = -X negates the odd coefficients
    sign = np.array([1 if t % 2 == 0 else -1 for t in range(N)], dtype=object)
    assert [int(x) for x in O.automorphism(a, N + 1)] == [int(x) * int(s) % Q for x, s in zip(a, sign)]


def _trace_setup(N, base_log, level, noiseless, seed):
    rs = np.random.default_rng(seed)
    S = (rs.integers(0, 2, size=N, dtype=np.uint64)).astype(np.uint64)
    steps = N.bit_length() - 1
    mask = rs.integers(0, 2**64, size=(steps, level, N), dtype=np.uint64, endpoint=False)
    noise = np.rint(rs.standard_normal((steps, level, N)) * 2.0 ** 13).astype(np.int64).view(np.uint64)
    if noiseless:
        mask[:] = 0
        noise[:] = 0
    return S, O.trace_keys(S, base_log, level, mask, noise)


@pytest.mark.parametrize("N", [16, 256])
def test_trace_noiseless_exact_gadget_closed_form(N):
    """Noiseless automorphism keys with a gadget covering all 64 bits (no
    rounding): the trace's phase is exactly N * phase[0] at coefficient 0
    and 0 elsewhere."""
    S, keys = _trace_setup(N, 16, 4, True, N)
    rs = random.Random(N + 7)
    c = rnd_u64(rs, 2 * N).reshape(1, 2, N)
    out = O.trace_batch(keys, c, 16, 4)
    ph_in = O.glwe_phase(S.reshape(1, N), c[0])
    ph_out = O.glwe_phase(S.reshape(1, N), out[0])
    assert int(ph_out[0]) == (N * int(ph_in[0])) % Q
    assert not ph_out[1:].any()


def test_trace_real_keys_isolates_constant_term():
    """Real (masked, noisy) keys: phase(Tr(c)) = N * phase(c)[0] at
    coefficient 0 and ~0 elsewhere, within the accumulated rounding and key
    noise of log2 N key switches."""
    N, bl, lv = 256, 8, 4
    S, keys = _trace_setup(N, bl, lv, False, 5)
    rs = np.random.default_rng(9)
    msg = (rs.integers(0, 16, size=N, dtype=np.uint64) << np.uint64(52)).astype(np.uint64)
    c = O.glwe_encrypt(S.reshape(1, N), msg, rs.integers(0, 2**64, size=(1, N), dtype=np.uint64, endpoint=False),
                       np.zeros(N, np.uint64)).reshape(1, 2, N)
    out = O.trace_batch(keys, c, bl, lv)
    ph = O.glwe_phase(S.reshape(1, N), out[0]).astype(object)
    want = [(N * int(msg[0])) % Q] + [0] * (N - 1)
    err = [((int(a) - b + Q // 2) % Q) - Q // 2 for a, b in zip(ph, want)]
    # per step: decomposition rounding (< 2^(63 - bl*lv) per coefficient times |S| <= N)
    # plus key noise (|d| <= 2^(bl-1), N lv terms of 6 sigma); the trace doubles what came before
    steps = N.bit_length() - 1
    per_step = N * (1 << (63 - bl * lv)) + N * lv * (1 << (bl - 1)) * 6 * (1 << 13)
    bound = per_step * (2 ** steps)
    assert max(abs(e) for e in err) < bound
    assert bound < (1 << 52) * N // 2     # the bound itself leaves the message readable


# ------------------------------------------------------------------ plaintext x ciphertext

@pytest.mark.parametrize("N", [1, 4, 16])
def test_plaintext_mul_matches_integer_convolution(N):
    """(P * A, P * B + Q) with P signed: each component an exact integer
    negacyclic convolution reduced mod 2^64 (the linear mapping of the
    lookup protocol, Cryptographic Lookup Protocol, Steps 2 and 3)."""
    rs = random.Random(100 + N)
    for with_q in (False, True):
        P = [rs.randrange(-2**63, 2**63) for _ in range(N)]
        c = [[rs.getrandbits(64) for _ in range(N)] for _ in range(2)]
        q = [rs.getrandbits(64) for _ in range(N)]
        want = []
        for comp in range(2):
            w = [0] * N
            for i in range(N):
                for j in range(N):
                    t = i + j
                    w[t % N] += (P[i] * c[comp][j]) * (-1 if t >= N else 1)
            if comp == 1 and with_q:
                w = [w[t] + q[t] for t in range(N)]
            want.append([x % Q for x in w])
        got = O.plaintext_mul_batch(np.array([c], np.uint64), np.array(P, np.int64),
                                    np.array(q, np.uint64) if with_q else None)
        assert [[int(x) for x in row] for row in got[0]] == want


def test_plaintext_mul_scales_the_phase():
    """phase(P * c) = P * phase(c): the product by a plaintext acts on the
    encrypted message (noiseless encryption of m under S)."""
    N = 64
    g = np.random.default_rng(5)
    S = g.integers(0, 2, size=(1, N), dtype=np.uint64)
    A = g.integers(0, 2**64, size=(1, N), dtype=np.uint64, endpoint=False)
    m = (g.integers(0, 16, size=N, dtype=np.uint64) << np.uint64(58))
    glwe = O.glwe_encrypt(S, m, A, np.zeros(N, np.uint64))
    P = g.integers(-3, 4, size=N)
    got = O.plaintext_mul_batch(glwe.reshape(1, 2, N), P)[0]
    ph = O.glwe_phase(S, got)
    # P * m by hand: negacyclic, small P
    want = [0] * N
    for i in range(N):
        for j in range(N):
            t = i + j
            want[t % N] += int(P[i]) * int(m[j]) * (-1 if t >= N else 1)
    assert [int(x) for x in ph] == [x % Q for x in want]


@pytest.mark.parametrize("N,base_log,level", [(64, 28, 2), (128, 16, 4), (64, 21, 3), (256, 9, 7)])
@pytest.mark.parametrize("sign", [+1, -1])
def test_cmux_at_the_largest_magnitude_closed_form(N, base_log, level, sign):
    """One CMux with a~ = N on a GLWE of constant C/2: every digit of the
    CMux input is -B/2 (closed form of the balanced decomposition), so the
    rotated GLWE is C/2 plus -B/2 times the negacyclic running sums of the
    key words -- every coefficient known without the oracle's arithmetic."""
    from tests import extreme_util as X
    p = W.Params("extreme", n=2, k=1, N=N, pbs_base_log=base_log, pbs_level=level, ks_base_log=4, ks_level=4,
                 msg_bits=3, lwe_sigma_log2=40, glwe_sigma_log2=20, lut=("square_mod",), msg=("uniform",),
                 batch=1, seed=1)
    bsk, lwe, glwe, C = X.case(p, sign, seed=N + level)
    got = O.blind_rotate_glwe_batch(p, bsk, lwe, glwe)
    want, peak = X.expected(p, bsk, C)
    assert peak > 1 << (62 + base_log)
    assert [[int(w) for w in row] for row in got[0]] == want
