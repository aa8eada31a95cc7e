"""GPU parity of the widened entry points: a LUT per ciphertext (many LUTs
in one launch) and blind rotation of encrypted (GLWE) test polynomials.
Bit-exact against the CPU oracle."""

import numpy as np
import pytest

import oracle as O
import workload as W
from tests import gpu_util as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_16915_gb300 import build
    build.build()


def _index_dev(idx):
    import torch
    return torch.from_numpy(np.asarray(idx, dtype=np.int32)).cuda()


def test_multi_lut_bitexact_and_decrypts():
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p))
    tables = [[(m * m) % 8 for m in range(8)], [(3 * m + 1) % 8 for m in range(8)], [7 - m for m in range(8)]]
    luts = np.stack([W.lut_torus(p, codes=t) for t in tables])
    rs = np.random.default_rng(2)
    idx = rs.integers(0, 3, size=40)
    cd = W.cipher_draws(p, 40, sub=21)
    lwe = keys.encrypt(cd)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    out = G.empty_dev(40, p.n + 1)
    ctx.pbs_batch_multi_lut(G.to_dev(lwe), G.to_dev(luts), _index_dev(idx), out)
    ctx.sync_status()
    got = G.to_host(out)
    assert np.array_equal(got, O.pbs_batch_multi_lut(p, keys.bsk, keys.ksk, lwe, luts, idx))
    want_codes = np.array([tables[i][m] for i, m in zip(idx, cd.codes)])
    assert np.array_equal(keys.decrypt(got), want_codes)


def test_multi_lut_full_batch_sampled():
    """The benchmark's many-LUT launch: standard set, 4096 ciphertexts, four
    LUTs round-robin; sparse-mask inputs at seeded positions are checked
    word for word, the rest are dense uniform words."""
    p = W.CONFIGS["standard"]
    bsk, ksk = W.uniform_keys(p, seed=61)
    codes = W.lut_codes(p)
    luts = np.stack([W.lut_torus(p, np.roll(codes, r)) for r in range(4)])
    idx = np.arange(p.batch) % 4
    lwe = W.uniform_ciphertexts(p, p.batch, sub=62)
    pos = np.array([0, 1, 2, 3, p.batch - 1])
    lwe[pos] = G.sparse_lwe(p, len(pos), 2, seed=63)
    ctx = G.make_ctx(p, bsk, ksk, max_batch=p.batch)
    out = G.empty_dev(p.batch, p.n + 1)
    ctx.pbs_batch_multi_lut(G.to_dev(lwe), G.to_dev(luts), _index_dev(idx), out)
    ctx.sync_status()
    got = G.to_host(out)
    assert np.array_equal(got[pos], O.pbs_batch_multi_lut(p, bsk, ksk, lwe[pos], luts, idx[pos]))


def test_multi_lut_bad_index_is_reported_not_followed():
    import paper_2609_16915_gb300 as R
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p))
    luts = np.stack([W.lut_torus(p), W.lut_torus(p, codes=[1] * 8)])
    lwe = W.uniform_ciphertexts(p, 4, sub=22)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    out = G.empty_dev(4, p.n + 1)
    ctx.pbs_batch_multi_lut(G.to_dev(lwe), G.to_dev(luts), _index_dev([0, 1, 5, 1]), out)
    with pytest.raises(R.RosettaError) as e:
        ctx.sync_status()
    assert e.value.status == -1
    ctx.sync_status()                                   # the flag is cleared once reported
    got = G.to_host(out)
    want = O.pbs_batch_multi_lut(p, keys.bsk, keys.ksk, lwe, luts, [0, 1, 0, 1])
    assert np.array_equal(got, want)


@pytest.mark.parametrize("name", ["tiny", "standard"])
def test_glwe_blind_rotation_bitexact(name):
    p = W.CONFIGS[name]
    if name == "tiny":
        keys = O.Keys(p, W.key_draws(p))
        bsk, ksk = keys.bsk, keys.ksk
        lwe = keys.encrypt(W.cipher_draws(p, 9, sub=23))
    else:
        bsk, ksk = W.uniform_keys(p, seed=31)
        lwe = G.sparse_lwe(p, 3, 2, seed=4)
    glwe = W.uniform_u64((lwe.shape[0], p.k + 1, p.N), W.rng(p.seed, "sample", 24))
    ctx = G.make_ctx(p, bsk, ksk)
    out = G.empty_dev(lwe.shape[0], p.k + 1, p.N)
    ctx.blind_rotate_glwe_batch(G.to_dev(lwe), G.to_dev(glwe), out)
    ctx.sync_status()
    assert np.array_equal(G.to_host(out), O.blind_rotate_glwe_batch(p, bsk, lwe, glwe))


def test_glwe_blind_rotation_trivial_input_matches_pbs_path():
    """A trivial GLWE of the test polynomial through the GLWE entry point,
    then extraction and key switch, gives rosetta_pbs_batch's words."""
    p = W.CONFIGS["standard"]
    bsk, ksk = W.uniform_keys(p, seed=32)
    lwe = G.sparse_lwe(p, 2, 3, seed=6)
    lut = W.lut_torus(p)
    glwe = np.zeros((2, p.k + 1, p.N), np.uint64)
    glwe[:, p.k] = O.test_poly(lut, p.msg_bits, p.N)
    ctx = G.make_ctx(p, bsk, ksk)
    out = G.empty_dev(2, p.k + 1, p.N)
    ctx.blind_rotate_glwe_batch(G.to_dev(lwe), G.to_dev(glwe), out)
    ctx.sync_status()
    acc = G.to_host(out)
    big = np.stack([O.sample_extract(acc[b]) for b in range(2)])
    assert np.array_equal(G.gpu_keyswitch(ctx, p, big), G.gpu_pbs(ctx, p, lwe, lut))


def test_glwe_blind_rotation_rejects_host_buffers():
    import paper_2609_16915_gb300 as R
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p))
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    lwe = W.uniform_ciphertexts(p, 2)
    glwe = np.zeros((2, p.k + 1, p.N), np.uint64)
    with pytest.raises(R.RosettaError) as e:
        ctx.blind_rotate_glwe_batch(lwe, glwe, np.zeros_like(glwe))
    assert e.value.status == -1


# ------------------------------------------------------------------ RLWE trace

def _trace_keys(p, base_log, level, noiseless, seed):
    g = np.random.default_rng(seed)
    S = g.integers(0, 2, size=p.N, dtype=np.uint64)
    steps = p.N.bit_length() - 1
    mask = g.integers(0, 2**64, size=(steps, level, p.N), dtype=np.uint64, endpoint=False)
    noise = np.rint(g.standard_normal((steps, level, p.N)) * 2.0 ** 13).astype(np.int64).view(np.uint64)
    if noiseless:
        mask[:] = 0
        noise[:] = 0
    return S, O.trace_keys(S, base_log, level, mask, noise)


@pytest.mark.parametrize("name,base_log,level", [("tiny", 16, 4), ("standard", 12, 4), ("gpt2_mlp", 16, 2)])
def test_trace_bitexact(name, base_log, level):
    """GPU trace word for word against the oracle (random keys and inputs)."""
    p = W.CONFIGS[name]
    S, keys = _trace_keys(p, base_log, level, False, 3)
    glwe = W.uniform_u64((5, 2, p.N), W.rng(p.seed, "sample", 41))
    import paper_2609_16915_gb300 as R
    ctx = R.Context(p)
    ctx.upload_trace_keys(G.to_dev(keys), base_log, level)
    out = G.empty_dev(5, 2, p.N)
    ctx.trace_batch(G.to_dev(glwe), out)
    ctx.sync_status()
    assert np.array_equal(G.to_host(out), O.trace_batch(keys, glwe, base_log, level))


def test_trace_noiseless_closed_form_on_gpu():
    """Noiseless keys, gadget over all 64 bits: phase(out) = (N phase(in)[0], 0, ..)."""
    p = W.CONFIGS["standard"]
    S, keys = _trace_keys(p, 16, 4, True, 4)
    glwe = W.uniform_u64((3, 2, p.N), W.rng(p.seed, "sample", 42))
    import paper_2609_16915_gb300 as R
    ctx = R.Context(p)
    ctx.upload_trace_keys(G.to_dev(keys), 16, 4)
    out = G.empty_dev(3, 2, p.N)
    ctx.trace_batch(G.to_dev(glwe), out)
    ctx.sync_status()
    got = G.to_host(out)
    for b in range(3):
        ph_in = O.glwe_phase(S.reshape(1, -1), glwe[b])
        ph = O.glwe_phase(S.reshape(1, -1), got[b])
        assert int(ph[0]) == (p.N * int(ph_in[0])) % (1 << 64)
        assert not ph[1:].any()


def test_trace_argument_checks():
    import paper_2609_16915_gb300 as R
    p = W.CONFIGS["standard"]
    ctx = R.Context(p)
    glwe = G.to_dev(np.zeros((1, 2, p.N), np.uint64))
    with pytest.raises(R.RosettaError) as e:
        ctx.trace_batch(glwe, G.empty_dev(1, 2, p.N))
    assert e.value.status == -3                     # keys missing
    keys = np.zeros((11, 3, 2, p.N), np.uint64)
    with pytest.raises(R.RosettaError) as e:
        ctx.upload_trace_keys(G.to_dev(keys), 16, 3)   # odd level
    assert e.value.status == -2
    big = R.Context(W.CONFIGS["llama_silu"])
    with pytest.raises(R.RosettaError) as e:
        big.upload_trace_keys(G.to_dev(np.zeros((13, 2, 2, 8192), np.uint64)), 16, 2)
    assert e.value.status == -2                     # N = 8192 not supported for the trace


# ------------------------------------------------------------------ plaintext x ciphertext

@pytest.mark.parametrize("name,batch,full_range,with_q", [
    ("tiny", 7, True, True), ("standard", 5, True, False), ("standard", 3, False, True), ("gpt2_mlp", 3, True, True)])
def test_plaintext_mul_bitexact(name, batch, full_range, with_q):
    """(P * A, P * B + Q) word for word against the oracle; P over all of int64
    or small, Q random or absent, a ragged batch."""
    p = W.CONFIGS[name]
    g = np.random.default_rng(batch + p.N)
    if full_range:
        P = g.integers(-2**63, 2**63, size=p.N, dtype=np.int64)
    else:
        P = g.integers(-1000, 1001, size=p.N, dtype=np.int64)
    Qv = W.uniform_u64((p.N,), W.rng(p.seed, "sample", 61)) if with_q else None
    glwe = W.uniform_u64((batch, 2, p.N), W.rng(p.seed, "sample", 60))
    import paper_2609_16915_gb300 as R
    ctx = R.Context(p)
    out = G.empty_dev(batch, 2, p.N)
    ctx.plaintext_mul_batch(G.to_dev(glwe), P, out, plain_add=Qv)
    ctx.sync_status()
    assert np.array_equal(G.to_host(out), O.plaintext_mul_batch(glwe, P, Qv))


def test_plaintext_mul_device_q_and_reuse():
    """Q from device memory; a second call with another P reuses the staged rows."""
    p = W.CONFIGS["standard"]
    g = np.random.default_rng(9)
    glwe = W.uniform_u64((2, 2, p.N), W.rng(p.seed, "sample", 62))
    Qv = W.uniform_u64((p.N,), W.rng(p.seed, "sample", 63))
    import paper_2609_16915_gb300 as R
    ctx = R.Context(p)
    for _ in range(2):
        P = g.integers(-2**20, 2**20, size=p.N, dtype=np.int64)
        out = G.empty_dev(2, 2, p.N)
        ctx.plaintext_mul_batch(G.to_dev(glwe), P, out, plain_add=G.to_dev(Qv))
        ctx.sync_status()
        assert np.array_equal(G.to_host(out), O.plaintext_mul_batch(glwe, P, Qv))


def test_plaintext_mul_argument_checks():
    import paper_2609_16915_gb300 as R
    p = W.CONFIGS["standard"]
    ctx = R.Context(p)
    P = np.zeros(p.N, np.int64)
    with pytest.raises(R.RosettaError) as e:        # host ciphertexts
        ctx.plaintext_mul_batch(np.zeros((1, 2, p.N), np.uint64), P, G.empty_dev(1, 2, p.N))
    assert e.value.status == -1
    with pytest.raises(R.RosettaError) as e:        # device P
        ctx.plaintext_mul_batch(G.to_dev(np.zeros((1, 2, p.N), np.uint64)), G.to_dev(P.view(np.uint64)),
                                G.empty_dev(1, 2, p.N))
    assert e.value.status == -1
    big = R.Context(W.CONFIGS["llama_silu"])
    N8 = W.CONFIGS["llama_silu"].N
    with pytest.raises(R.RosettaError) as e:
        big.plaintext_mul_batch(G.to_dev(np.zeros((1, 2, N8), np.uint64)), np.zeros(N8, np.int64),
                                G.empty_dev(1, 2, N8))
    assert e.value.status == -2


# ------------------------------------------------------------------ encrypted segmented lookup

def _lookup_ctx(p, bsk, ksk, tk, tb, tl, tables):
    ctx = G.make_ctx(p, bsk, ksk)
    ctx.upload_trace_keys(G.to_dev(tk), tb, tl)
    ctx.upload_lookup_table(*tables)
    return ctx


def test_lookup_bitexact_and_decrypts_small_ring():
    """Real keys, the paper's 1/x table: GPU words = oracle words, and the
    decryption is the cleartext segmented lookup (4.571 at x = 0.22)."""
    from paper_2609_16915_gb300 import segmented as SG
    from tests import lookup_util as LU
    p = W.CONFIGS["lookup_small"]
    keys = O.Keys(p, W.key_draws(p))
    tk = LU.trace_keys(p, keys.glwe_key)
    lut = LU.paper_table()
    enc = SG.encode(lut, p.N, LU.DX, LU.DR)
    xs = [0.22] + LU.sample_points(lut, 8, 11)
    segs = [SG.segment_index(lut, x) for x in xs]
    glwe, lwe = LU.encrypt_inputs(p, keys, xs, segs, lut.n_seg, sub=1)
    tables = (enc.p_hat, enc.q_hat, enc.a_hat, enc.b_hat)
    ctx = _lookup_ctx(p, keys.bsk, keys.ksk, tk, LU.TRACE_BASE_LOG, LU.TRACE_LEVEL, tables)
    out = G.empty_dev(len(xs), 2, p.N)
    ctx.segmented_lookup_batch(G.to_dev(glwe), G.to_dev(lwe), out)
    ctx.sync_status()
    got = G.to_host(out)
    want = O.segmented_lookup_batch(p, keys.bsk, keys.ksk, tk, LU.TRACE_BASE_LOG, LU.TRACE_LEVEL, glwe, lwe, *tables)
    assert np.array_equal(got, want)
    S = keys.glwe_key.reshape(1, -1)
    vals = [SG.decode(O.glwe_phase(S, got[b])[0], enc) for b in range(len(xs))]
    # the running example's value (4.571 printed) within the noise of the
    # encrypted path: about 1.2e-3 standard deviation at these parameters
    assert round(SG.lookup(lut, 0.22), 3) == 4.571
    assert vals[0] == pytest.approx(SG.lookup(lut, 0.22), abs=6e-3)
    for x, v in zip(xs, vals):
        assert v == pytest.approx(SG.lookup(lut, x), abs=1e-2), x


@pytest.mark.parametrize("n_seg", [1, 8])
def test_lookup_bitexact_random_tables(n_seg):
    """Random integer tables and uniform-word keys and inputs, other segment counts."""
    p = W.CONFIGS["lookup_small"]
    g = np.random.default_rng(40 + n_seg)
    bsk, ksk = W.uniform_keys(p, seed=41)
    tk = W.uniform_u64((p.N.bit_length() - 1, 4, 2, p.N), W.rng(p.seed, "sample", 80))
    tables = (g.integers(-2**40, 2**40, size=p.N, dtype=np.int64), W.uniform_u64((p.N,), W.rng(p.seed, "sample", 81)),
              g.integers(-2**40, 2**40, size=(n_seg, p.N), dtype=np.int64),
              W.uniform_u64((n_seg, p.N), W.rng(p.seed, "sample", 82)))
    glwe = W.uniform_u64((3, 2, p.N), W.rng(p.seed, "sample", 83))
    lwe = W.uniform_u64((3, p.n + 1), W.rng(p.seed, "sample", 84))
    ctx = _lookup_ctx(p, bsk, ksk, tk, 16, 4, tables)
    out = G.empty_dev(3, 2, p.N)
    ctx.segmented_lookup_batch(G.to_dev(glwe), G.to_dev(lwe), out)
    ctx.sync_status()
    assert np.array_equal(G.to_host(out), O.segmented_lookup_batch(p, bsk, ksk, tk, 16, 4, glwe, lwe, *tables))


def test_lookup_bitexact_standard_ring():
    """N = 2048, n = 742 (the bench's ring): one ciphertext, four segments,
    sparse segment-index ciphertext (the oracle's cost)."""
    p = W.CONFIGS["standard"]
    g = np.random.default_rng(50)
    bsk, ksk = W.uniform_keys(p, seed=51)
    tk = W.uniform_u64((p.N.bit_length() - 1, 4, 2, p.N), W.rng(p.seed, "sample", 90))
    n_seg = 4
    tables = (g.integers(-2**40, 2**40, size=p.N, dtype=np.int64), W.uniform_u64((p.N,), W.rng(p.seed, "sample", 91)),
              g.integers(-2**40, 2**40, size=(n_seg, p.N), dtype=np.int64),
              W.uniform_u64((n_seg, p.N), W.rng(p.seed, "sample", 92)))
    glwe = W.uniform_u64((1, 2, p.N), W.rng(p.seed, "sample", 93))
    lwe = G.sparse_lwe(p, 1, 3, seed=9)
    ctx = _lookup_ctx(p, bsk, ksk, tk, 16, 4, tables)
    out = G.empty_dev(1, 2, p.N)
    ctx.segmented_lookup_batch(G.to_dev(glwe), G.to_dev(lwe), out)
    ctx.sync_status()
    assert np.array_equal(G.to_host(out), O.segmented_lookup_batch(p, bsk, ksk, tk, 16, 4, glwe, lwe, *tables))


def test_lookup_full_batch_sampled():
    """The benchmark's lookup launch: standard ring, 1024 ciphertexts, four
    segments, trace gadget 2^16 x 4; two seeded positions (sparse segment
    index ciphertexts, for the oracle's cost) are checked word for word."""
    p = W.CONFIGS["standard"]
    g = np.random.default_rng(70)
    batch, n_seg = 1024, 4
    bsk, ksk = W.uniform_keys(p, seed=71)
    tk = W.uniform_u64((p.N.bit_length() - 1, 4, 2, p.N), W.rng(p.seed, "sample", 72))
    tables = (g.integers(-2**40, 2**40, size=p.N, dtype=np.int64), W.uniform_u64((p.N,), W.rng(p.seed, "sample", 73)),
              g.integers(-2**40, 2**40, size=(n_seg, p.N), dtype=np.int64),
              W.uniform_u64((n_seg, p.N), W.rng(p.seed, "sample", 74)))
    glwe = W.uniform_u64((batch, 2, p.N), W.rng(p.seed, "sample", 75))
    lwe = W.uniform_ciphertexts(p, batch, sub=76)
    pos = np.array([0, batch - 1])
    lwe[pos] = G.sparse_lwe(p, len(pos), 3, seed=77)
    ctx = _lookup_ctx(p, bsk, ksk, tk, 16, 4, tables)
    out = G.empty_dev(batch, 2, p.N)
    ctx.segmented_lookup_batch(G.to_dev(glwe), G.to_dev(lwe), out)
    ctx.sync_status()
    got = G.to_host(out)
    want = O.segmented_lookup_batch(p, bsk, ksk, tk, 16, 4, glwe[pos], lwe[pos], *tables)
    assert np.array_equal(got[pos], want)


def test_lookup_argument_checks():
    import paper_2609_16915_gb300 as R
    p = W.CONFIGS["lookup_small"]
    bsk, ksk = W.uniform_keys(p, seed=42)
    ctx = G.make_ctx(p, bsk, ksk)
    glwe = G.to_dev(np.zeros((1, 2, p.N), np.uint64))
    lwe = G.to_dev(np.zeros((1, p.n + 1), np.uint64))
    with pytest.raises(R.RosettaError) as e:        # no trace keys, no tables
        ctx.segmented_lookup_batch(glwe, lwe, G.empty_dev(1, 2, p.N))
    assert e.value.status == -3
    z64, zu = np.zeros(p.N, np.int64), np.zeros(p.N, np.uint64)
    with pytest.raises(R.RosettaError) as e:        # 3 segments: not a power of two
        ctx.upload_lookup_table(z64, zu, np.zeros((3, p.N), np.int64), np.zeros((3, p.N), np.uint64))
    assert e.value.status == -2
    with pytest.raises(R.RosettaError) as e:        # tables in device memory
        ctx.upload_lookup_table(G.to_dev(zu), zu, np.zeros((2, p.N), np.int64), np.zeros((2, p.N), np.uint64))
    assert e.value.status == -1


def test_lookup_one_interval_per_coefficient_on_gpu():
    """N_br = N (boxes of one coefficient, the paper's setting): GPU words =
    oracle words, decrypting to the cleartext lookup."""
    from paper_2609_16915_gb300 import segmented as SG
    from tests import lookup_util as LU
    p = W.CONFIGS["lookup_small"]
    keys = O.Keys(p, W.key_draws(p))
    tk = LU.trace_keys(p, keys.glwe_key)
    lut = SG.build(SG.FUNCTIONS["reciprocal"], [0.1, 0.5, 2.0], p.N)
    enc = SG.encode(lut, p.N, LU.DX, LU.DR)
    xs = LU.sample_points(lut, 8, 19)
    segs = [SG.segment_index(lut, x) for x in xs]
    glwe, lwe = LU.encrypt_inputs(p, keys, xs, segs, lut.n_seg, sub=4)
    tables = (enc.p_hat, enc.q_hat, enc.a_hat, enc.b_hat)
    ctx = _lookup_ctx(p, keys.bsk, keys.ksk, tk, LU.TRACE_BASE_LOG, LU.TRACE_LEVEL, tables)
    out = G.empty_dev(len(xs), 2, p.N)
    ctx.segmented_lookup_batch(G.to_dev(glwe), G.to_dev(lwe), out)
    ctx.sync_status()
    got = G.to_host(out)
    assert np.array_equal(got, O.segmented_lookup_batch(p, keys.bsk, keys.ksk, tk, LU.TRACE_BASE_LOG,
                                                        LU.TRACE_LEVEL, glwe, lwe, *tables))
    S = keys.glwe_key.reshape(1, -1)
    for b, x in enumerate(xs):
        assert SG.decode(O.glwe_phase(S, got[b])[0], enc) == pytest.approx(SG.lookup(lut, x), abs=1e-2)
