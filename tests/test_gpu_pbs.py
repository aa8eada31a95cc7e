"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Integer work, so the bar is bit-exact equality of every output word.  Small
cases compare every ciphertext; full-size launches (the batch sizes the
benchmark times) compare a seeded sample with the oracle and check the rest
by decryption.  Sparse-mask inputs make blind rotation run only a few CMux
steps, which lets the oracle check the largest parameter sets quickly."""

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
    import paper_2609_16915_gb300 as R
    R.load()


_KEYS = {}


def torch_device_count():
    import torch
    return torch.cuda.device_count()


def real_keys(name):
    if name not in _KEYS:
        p = W.CONFIGS[name]
        _KEYS[name] = O.Keys(p, W.key_draws(p))
    return _KEYS[name]


# ------------------------------------------------------------------ tiny

@pytest.mark.parametrize("batch", [1, 16, 37])
def test_tiny_pbs_bitexact_and_decrypts(batch):
    p = W.CONFIGS["tiny"]
    keys = real_keys("tiny")
    cd = W.cipher_draws(p, batch, sub=batch)
    lwe = keys.encrypt(cd)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    got = G.gpu_pbs(ctx, p, lwe, lut)
    want = O.pbs_batch(p, keys.bsk, keys.ksk, lwe, lut)
    assert np.array_equal(got, want)
    assert np.array_equal(keys.decrypt(got), W.lut_codes(p)[cd.codes])


def test_tiny_stagewise_blind_rotate_then_keyswitch():
    p = W.CONFIGS["tiny"]
    keys = real_keys("tiny")
    lwe = W.uniform_ciphertexts(p, 24, sub=3)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    big = G.gpu_br_extract(ctx, p, lwe, lut)
    want_big = O.blind_rotate_extract_batch(p, keys.bsk, lwe, lut)
    assert np.array_equal(big, want_big)
    ks = G.gpu_keyswitch(ctx, p, want_big)
    assert np.array_equal(ks, O.keyswitch_batch(p, keys.ksk, want_big))


def test_tiny_noiseless_keys_closed_form():
    """With zero-mask, zero-noise keys the PBS output is (0,..,0, F(m~)), the
    negacyclic LUT at the modulus-switched phase (same closed form the oracle
    is pinned to)."""
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p, trivial=True))
    lut = W.lut_torus(p, codes=[(5 * m + 3) % 8 for m in range(8)])
    lwe = W.uniform_ciphertexts(p, 40, sub=9)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    got = G.gpu_pbs(ctx, p, lwe, lut)
    assert np.array_equal(got, O.pbs_batch(p, keys.bsk, keys.ksk, lwe, lut))
    assert not got[:, :p.n].any()


# ------------------------------------------------------------------ every ring size, single CMux steps

SIZES = {
    256: W.CONFIGS["tiny"],
    512: W.Params("n512", n=100, k=1, N=512, pbs_base_log=12, pbs_level=2, ks_base_log=4, ks_level=4, msg_bits=4,
                  lwe_sigma_log2=40, glwe_sigma_log2=20, lut=("square_mod",), msg=("uniform",), batch=8, seed=11),
    1024: W.Params("n1024", n=300, k=1, N=1024, pbs_base_log=20, pbs_level=1, ks_base_log=3, ks_level=5, msg_bits=4,
                   lwe_sigma_log2=40, glwe_sigma_log2=20, lut=("square_mod",), msg=("uniform",), batch=8, seed=12),
    2048: W.CONFIGS["standard"],
    4096: W.CONFIGS["gpt2_mlp"],
    8192: W.CONFIGS["llama_silu"],
}


@pytest.mark.parametrize("N", sorted(SIZES))
def test_sparse_blind_rotation_every_size(N):
    """Uniform-word keys (what real keys look like) and inputs with 1-3
    nonzero mask words: every ring size and gadget the kernels instantiate."""
    p = SIZES[N]
    bsk, ksk = W.uniform_keys(p, seed=100 + N)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, bsk, ksk)
    lwe = np.concatenate([G.sparse_lwe(p, 2, 1, seed=N), G.sparse_lwe(p, 2, 3, seed=N + 1)])
    got = G.gpu_br_extract(ctx, p, lwe, lut)
    want = O.blind_rotate_extract_batch(p, bsk, lwe, lut)
    assert np.array_equal(got, want)
    got_pbs = G.gpu_pbs(ctx, p, lwe[:2], lut)
    assert np.array_equal(got_pbs, O.keyswitch_batch(p, ksk, want[:2]))


# ------------------------------------------------------------------ standard / full-size launches

def test_standard_dense_bitexact():
    p = W.CONFIGS["standard"]
    keys = real_keys("standard")
    cd = W.cipher_draws(p, 20, sub=1)
    lwe = keys.encrypt(cd)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    got = G.gpu_pbs(ctx, p, lwe, lut)
    sample = np.arange(0, 20, 2)
    want = O.pbs_batch(p, keys.bsk, keys.ksk, lwe[sample], lut)
    assert np.array_equal(got[sample], want)
    assert np.array_equal(keys.decrypt(got), W.lut_codes(p)[cd.codes])


def test_standard_full_batch_sampled():
    """The benchmark's launch: 4096 ciphertexts in one call; a seeded sample
    is checked word for word, all of them by decryption."""
    p = W.CONFIGS["standard"]
    keys = real_keys("standard")
    cd = W.cipher_draws(p, p.batch, sub=2)
    lwe = keys.encrypt(cd)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk, max_batch=p.batch)
    got = G.gpu_pbs(ctx, p, lwe, lut)
    sample = np.random.default_rng(7).choice(p.batch, size=6, replace=False)
    sample[0], sample[1] = 0, p.batch - 1
    assert np.array_equal(got[sample], O.pbs_batch(p, keys.bsk, keys.ksk, lwe[sample], lut))
    fails = int(np.sum(keys.decrypt(got) != W.lut_codes(p)[cd.codes]))
    assert fails == 0


@pytest.mark.parametrize("batch", [1, 64, 1024])
def test_exp_sweep_batches(batch):
    p = W.CONFIGS["exp_sweep"]
    keys = O.Keys(p, W.key_draws(p))
    cd = W.cipher_draws(p, batch, sub=batch)
    lwe = keys.encrypt(cd)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    got = G.gpu_pbs(ctx, p, lwe, lut)
    sample = np.unique(np.array([0, batch - 1, batch // 2]))
    assert np.array_equal(got[sample], O.pbs_batch(p, keys.bsk, keys.ksk, lwe[sample], lut))
    # the 5-bit exp LUT has a thin noise margin; failures are reported, a few are expected
    fails = int(np.sum(keys.decrypt(got) != W.lut_codes(p)[cd.codes]))
    assert fails <= max(2, batch // 100)


@pytest.mark.parametrize("batch", [16384, 65536])
def test_exp_sweep_large_batches_sampled(batch):
    """The sweep's two largest launches: a seeded sample word for word, the
    whole batch by decryption (the 5-bit exp LUT's thin margin allows a few
    failures)."""
    p = W.CONFIGS["exp_sweep"]
    keys = real_keys("exp_sweep")
    cd = W.cipher_draws(p, batch, sub=batch)
    lwe = keys.encrypt(cd)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk, max_batch=batch)
    got = G.gpu_pbs(ctx, p, lwe, lut)
    sample = np.array([0, batch // 2, batch - 1])
    assert np.array_equal(got[sample], O.pbs_batch(p, keys.bsk, keys.ksk, lwe[sample], lut))
    fails = int(np.sum(keys.decrypt(got) != W.lut_codes(p)[cd.codes]))
    assert fails <= batch // 100


@pytest.mark.parametrize("name", ["gpt2_mlp", "llama_silu"])
def test_large_configs_full_batch_sparse_sample(name):
    """Full-size launches of the two large parameter sets with uniform-word
    keys; the inputs at seeded positions are sparse so the oracle can check
    them, the others are dense uniform words."""
    p = W.CONFIGS[name]
    bsk, ksk = W.uniform_keys(p)
    lut = W.lut_torus(p)
    lwe = W.uniform_ciphertexts(p, p.batch, sub=4)
    pos = np.array([0, 1, p.batch // 3, p.batch - 1])
    lwe[pos] = G.sparse_lwe(p, len(pos), 2, seed=5)
    ctx = G.make_ctx(p, bsk, ksk, max_batch=p.batch)
    got = G.gpu_pbs(ctx, p, lwe, lut)
    want = O.keyswitch_batch(p, ksk, O.blind_rotate_extract_batch(p, bsk, lwe[pos], lut))
    assert np.array_equal(got[pos], want)


# ------------------------------------------------------------------ edge cases

def test_edge_inputs_match_oracle():
    """Zero masks (no CMux step runs), masks whose switched value is N (a
    pure negation), b~ = 0 and b~ = 2N-1, all-zero and constant LUTs."""
    p = W.CONFIGS["standard"]
    bsk, ksk = W.uniform_keys(p, seed=77)
    ctx = G.make_ctx(p, bsk, ksk)
    lwe = np.zeros((6, p.n + 1), np.uint64)
    lwe[1, :] = np.uint64(1 << 63)                     # every a~ = N, b~ = N
    lwe[2, 5] = np.uint64(1 << 63)
    lwe[3, p.n] = np.uint64(2**64 - 1)                  # b~ rounds to 0 (wraps)
    lwe[4, p.n] = np.uint64((2**64 - 1) - (1 << 51))    # b~ = 2N - 1
    lwe[5, 3] = np.uint64(1 << 51)                      # a~ = 1 (half-way tie rounds up)
    for lut in [W.lut_torus(p), np.zeros(16, np.uint64), np.full(16, 1 << 59, np.uint64)]:
        got = G.gpu_pbs(ctx, p, lwe, lut)
        want = O.keyswitch_batch(p, ksk, O.blind_rotate_extract_batch(p, bsk, lwe, lut))
        assert np.array_equal(got, want)


def test_keyswitch_ragged_tiles():
    """Batch and output width that are not multiples of the kernel's tiles."""
    p = W.CONFIGS["tiny"]
    keys = real_keys("tiny")
    rs = np.random.default_rng(3)
    big = rs.integers(0, 2**64, size=(101, p.kN + 1), dtype=np.uint64)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    assert np.array_equal(G.gpu_keyswitch(ctx, p, big), O.keyswitch_batch(p, keys.ksk, big))


def test_host_buffers_same_result():
    """The C ABI accepts host buffers (staged on the stream) as well."""
    p = W.CONFIGS["tiny"]
    keys = real_keys("tiny")
    lwe = W.uniform_ciphertexts(p, 19, sub=8)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    out = np.zeros((19, p.n + 1), np.uint64)
    ctx.pbs_batch(lwe, lut, out)
    assert np.array_equal(out, G.gpu_pbs(ctx, p, lwe, lut))
    assert np.array_equal(out, O.pbs_batch(p, keys.bsk, keys.ksk, lwe, lut))


def test_batch_zero_is_noop():
    p = W.CONFIGS["tiny"]
    keys = real_keys("tiny")
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    out = G.empty_dev(1, p.n + 1)
    out.fill_(7)
    ctx.pbs_batch(G.empty_dev(0, p.n + 1), G.to_dev(W.lut_torus(p)), out)
    ctx.sync_status()
    assert int(out[0, 0]) == 7


def test_error_codes():
    import ctypes
    import paper_2609_16915_gb300 as R
    L = R.load()
    p = W.CONFIGS["tiny"]
    # unsupported parameter sets
    for bad in [dict(N=128), dict(k=2), dict(pbs_base_log=29), dict(msg_bits=8)]:
        q = W.Params(**{**p.__dict__, **bad})
        with pytest.raises(R.RosettaError) as e:
            R.Context(q)
        assert e.value.status == -2
    ctx = R.Context(p)
    lwe = G.to_dev(W.uniform_ciphertexts(p, 4))
    lut = G.to_dev(W.lut_torus(p))
    out = G.empty_dev(4, p.n + 1)
    with pytest.raises(R.RosettaError) as e:      # keys missing
        ctx.pbs_batch(lwe, lut, out)
    assert e.value.status == -3
    keys = real_keys("tiny")
    ctx.upload_bsk(G.to_dev(keys.bsk))
    ctx.upload_ksk(G.to_dev(keys.ksk))
    with pytest.raises(R.RosettaError) as e:      # output aliases input
        ctx.pbs_batch(lwe, lut, lwe)
    assert e.value.status == -1
    st = L.rosetta_pbs_batch(ctx._h, None, 4, lut.data_ptr(), out.data_ptr(), None)
    assert st == -1
    st = L.rosetta_pbs_batch(ctx._h, lwe.data_ptr() + 4, 2, lut.data_ptr(), out.data_ptr(), None)
    assert st == -1                               # misaligned
    st = L.rosetta_upload_bsk(ctx._h, G.to_dev(keys.bsk).data_ptr(), keys.bsk.size - 1, 1, None)
    assert st == -1                               # wrong key size
    ctx.sync_status()
    small = G.make_ctx(p, keys.bsk, keys.ksk, max_batch=2)
    with pytest.raises(R.RosettaError) as e:      # batch above the context's max_batch
        small.pbs_batch(lwe, lut, out)
    assert e.value.status == -1
    got = G.gpu_pbs(small, p, W.uniform_ciphertexts(p, 2), W.lut_torus(p))
    assert got.shape == (2, p.n + 1)
    with pytest.raises(R.RosettaError) as e:      # no such device
        R.Context(p, device=torch_device_count() + 3)
    assert e.value.status == -4


def test_c_client_bootstraps_like_the_oracle(tmp_path):
    """A C99 program (tests/c_abi_demo.c) drives the library with host buffers:
    same words as the oracle."""
    import subprocess
    from tests.test_abi import build_c_client
    p = W.CONFIGS["tiny"]
    keys = real_keys("tiny")
    lwe = keys.encrypt(W.cipher_draws(p, 21, sub=31))
    lut = W.lut_torus(p)
    inp, outp = tmp_path / "in.bin", tmp_path / "out.bin"
    head = np.array([p.n, p.k, p.N, p.pbs_base_log, p.pbs_level, p.ks_base_log, p.ks_level, p.msg_bits, 0,
                     lwe.shape[0]], np.uint32)
    with open(inp, "wb") as f:
        for a in (head, keys.bsk, keys.ksk, lut, lwe):
            f.write(np.ascontiguousarray(a).tobytes())
    exe = build_c_client(str(tmp_path / "c_abi_demo"))
    r = subprocess.run([exe, str(inp), str(outp)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    got = np.fromfile(outp, dtype=np.uint64).reshape(lwe.shape)
    assert np.array_equal(got, O.pbs_batch(p, keys.bsk, keys.ksk, lwe, lut))
    assert np.array_equal(keys.decrypt(got), W.lut_codes(p)[W.cipher_draws(p, 21, sub=31).codes])
