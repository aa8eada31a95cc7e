"""Encrypted segmented lookup (Cryptographic Lookup Protocol, Steps 2 and 3):
the table encoder against the paper's printed polynomials, and the oracle's
composed lookup against a closed form and against the cleartext lookup
(itself pinned by the paper's running example)."""

import json
import os

import numpy as np
import pytest

import oracle as O
import workload as W
from paper_2609_16915_gb300 import segmented as SG
from tests import lookup_util as LU

G = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_segmented_example.json")))
Q = 1 << 64


def _signed(v):
    v = int(v) % Q
    return v - Q if v >= 1 << 63 else v


# ------------------------------------------------------------------ encoder

def test_encoder_carries_the_printed_index_polynomials():
    """Box centre s of p, q holds p_s, q_s of the example (10.0, 2.667; -1.0, -1.333)
    in units of Delta_I / Delta_x and Delta_I, q shifted by half an interval."""
    lut = LU.paper_table()
    N, DX = 256, 20
    enc = SG.encode(lut, N, DX, LU.DR)
    d_i = 2.0 ** (63 - 2)
    box = N // lut.n_seg
    for s in range(lut.n_seg):
        assert enc.p_hat[s * box] * 2.0 ** DX / d_i == pytest.approx(G["p_coeffs"][s], abs=2e-3)
        assert _signed(enc.q_hat[s * box]) / d_i + 0.5 == pytest.approx(G["q_coeffs"][s], abs=2e-3)
    # t = p x + q at the example point, box by box: the printed candidate indices
    x = G["x"]
    for s in range(lut.n_seg):
        t = (int(enc.p_hat[s * box]) * round(x * 2 ** DX) + _signed(enc.q_hat[s * box])) / d_i + 0.5
        assert t == pytest.approx(G["t"][s], abs=2e-3)


def test_encoder_carries_the_printed_value_polynomials():
    lut = LU.paper_table()
    N, DX = 256, 20
    enc = SG.encode(lut, N, DX, LU.DR)
    box = N // lut.n_br
    for i in range(lut.n_br):
        assert enc.a_hat[0][i * box] * 2.0 ** (DX - LU.DR) == pytest.approx(G["a0_coeffs"][i], abs=1e-2)
        assert _signed(enc.b_hat[0][i * box]) * 2.0 ** -LU.DR == pytest.approx(G["b0_coeffs"][i], abs=1e-2)
        # r_s at the example point, interval by interval
        for s, key in ((0, "r0"), (1, "r1")):
            r = (int(enc.a_hat[s][i * box]) * round(G["x"] * 2 ** DX) + _signed(enc.b_hat[s][i * box])) * 2.0 ** -LU.DR
            assert r == pytest.approx(G[key][i], abs=2e-3)


def test_box_layout_is_a_negacyclic_half_box_rotation():
    """Rotating the layout left by i boxes (X^-(i box)) puts values[i] on
    [-h, h) around 0 (the negacyclic wrap supplying the part below 0)."""
    N, vals = 64, [11, -7, 5, 3]
    lay = SG.box_layout(vals, N)
    box, h = N // len(vals), N // len(vals) // 2
    for i, v in enumerate(vals):
        rot = O.poly_monomial(np.array([x % Q for x in lay], np.uint64), (2 * N - i * box) % (2 * N))
        for d in range(-h, h):
            got = _signed(rot[d]) if d >= 0 else -_signed(rot[N + d])
            assert got == v, (i, d)


# ------------------------------------------------------------------ composed oracle

def _closed_form(N, n_seg, m_x, S, P, Qh, A, B):
    """Phase of the lookup output for trivial (noiseless, zero-mask) inputs:
    every blind rotation is the plain rotation by the input's modulus switch,
    every trace multiplies the constant coefficient by N and clears the rest."""
    log2_2N = (2 * N).bit_length() - 1
    sh = 64 - log2_2N

    def coef_after_rotation(poly, u):          # constant coefficient of X^-u poly
        u %= 2 * N
        return poly[u] % Q if u < N else (-poly[u - N]) % Q

    t = [(int(P[j]) * m_x + int(Qh[j])) % Q for j in range(N)]
    u_s = S * (N // n_seg)
    phi_i = coef_after_rotation(t, u_s)
    u_i = ((phi_i + (1 << (sh - 1))) >> sh) % (2 * N)
    vals = [int(A[S][j]) * m_x + int(B[S][j]) for j in range(N)]
    v = coef_after_rotation(vals, u_i)
    return (N * N * v) % Q


@pytest.mark.parametrize("n_seg", [1, 2, 4])
def test_composed_lookup_trivial_inputs_closed_form(n_seg):
    p = W.CONFIGS["tiny"]
    N = p.N
    g = np.random.default_rng(n_seg)
    keys = O.Keys(p, W.key_draws(p))
    tk = LU.trace_keys(p, keys.glwe_key, 16, 4)
    P = g.integers(-2**20, 2**20, size=N, dtype=np.int64)
    Qh = W.uniform_u64((N,), W.rng(1, "sample", 70))
    A = g.integers(-2**20, 2**20, size=(n_seg, N), dtype=np.int64)
    B = W.uniform_u64((n_seg, N), W.rng(1, "sample", 71))
    batch = 3
    xs = [int(v) for v in g.integers(-2**30, 2**30, size=batch)]
    Ss = [int(v) for v in g.integers(0, n_seg, size=batch)]
    glwe = np.zeros((batch, 2, N), np.uint64)
    lwe = np.zeros((batch, p.n + 1), np.uint64)
    for b in range(batch):
        glwe[b, 1, 0] = np.uint64(xs[b] % Q)
        lwe[b, -1] = np.uint64(SG.segment_word(Ss[b], n_seg))
    out = O.segmented_lookup_batch(p, keys.bsk, keys.ksk, tk, 16, 4, glwe, lwe, P, Qh, A, B)
    for b in range(batch):
        assert not out[b, 0].any()
        assert int(out[b, 1, 0]) == _closed_form(N, n_seg, xs[b], Ss[b], P, Qh, A, B)
        assert not out[b, 1, 1:].any()


@pytest.fixture(scope="module")
def small_setup():
    p = W.CONFIGS["lookup_small"]
    keys = O.Keys(p, W.key_draws(p))
    tk = LU.trace_keys(p, keys.glwe_key)
    lut = LU.paper_table()
    enc = SG.encode(lut, p.N, LU.DX, LU.DR)
    return p, keys, tk, lut, enc


def test_composed_lookup_decrypts_to_the_paper_value(small_setup):
    """Real keys: the encrypted lookup of the running example (x = 0.22) decrypts
    to a_01 x + b_01 = 4.571, and sampled points to the cleartext lookup."""
    p, keys, tk, lut, enc = small_setup
    xs = [G["x"]] + LU.sample_points(lut, 5, 7)
    segs = [SG.segment_index(lut, x) for x in xs]
    glwe, lwe = LU.encrypt_inputs(p, keys, xs, segs, lut.n_seg)
    out = O.segmented_lookup_batch(p, keys.bsk, keys.ksk, tk, LU.TRACE_BASE_LOG, LU.TRACE_LEVEL, glwe, lwe,
                                   enc.p_hat, enc.q_hat, enc.a_hat, enc.b_hat)
    S = keys.glwe_key.reshape(1, -1)
    got = [SG.decode(O.glwe_phase(S, out[b])[0], enc) for b in range(len(xs))]
    # within the noise of the encrypted path (about 1.2e-3 standard
    # deviation at these parameters) of the printed value
    assert got[0] == pytest.approx(G["value"], abs=6e-3)
    for x, v in zip(xs, got):
        assert v == pytest.approx(SG.lookup(lut, x), abs=1e-2), x


def test_composed_lookup_one_interval_per_coefficient(small_setup):
    """N_br = N (the paper's setting: every ring coefficient is an interval,
    boxes of one coefficient): the encrypted lookup still decrypts to the
    cleartext lookup, now with N intervals per segment."""
    p, keys, tk, _, _ = small_setup
    lut = SG.build(SG.FUNCTIONS["reciprocal"], [0.1, 0.5, 2.0], p.N)
    enc = SG.encode(lut, p.N, LU.DX, LU.DR)
    xs = LU.sample_points(lut, 6, 17)
    segs = [SG.segment_index(lut, x) for x in xs]
    glwe, lwe = LU.encrypt_inputs(p, keys, xs, segs, lut.n_seg, sub=3)
    out = O.segmented_lookup_batch(p, keys.bsk, keys.ksk, tk, LU.TRACE_BASE_LOG, LU.TRACE_LEVEL, glwe, lwe,
                                   enc.p_hat, enc.q_hat, enc.a_hat, enc.b_hat)
    S = keys.glwe_key.reshape(1, -1)
    for b, x in enumerate(xs):
        v = SG.decode(O.glwe_phase(S, out[b])[0], enc)
        assert v == pytest.approx(SG.lookup(lut, x), abs=1e-2), x
        # 512 intervals per segment: within the slope quantisation (2^-9 |x|) of 1/x
        assert v == pytest.approx(1.0 / x, abs=1e-2), x


@pytest.mark.parametrize("n_seg", [1, 2, 4, 8])
def test_oracle_segment_boxes_select_their_segment(n_seg):
    """Rotating the oracle's box polynomial of segment s left by s box + d
    (|d| within half a box, the noise a blind rotation by [[S]] can add)
    leaves 1 in the constant coefficient; its shift by another segment leaves 0."""
    N = 64
    box, h = N // n_seg, N // n_seg // 2
    for s in range(n_seg):
        b = np.array([x % Q for x in O.segment_box(s, n_seg, N).tolist()], np.uint64)
        for d in range(-h, box - h):
            rot = O.poly_monomial(b, (2 * N - (s * box + d)) % (2 * N))
            assert int(rot[0]) == 1, (s, d)
        for s2 in range(n_seg):
            if s2 != s:
                assert int(O.poly_monomial(b, (2 * N - s2 * box) % (2 * N))[0]) == 0
