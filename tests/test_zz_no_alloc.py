"""rosetta_pbs_batch_noalloc, the entry point for callers that cannot
allocate device memory during a call (device memory owned by another
allocator, or an allocation-free serving loop): it must return exactly what
rosetta_pbs_batch returns, call after call, even though every call reuses
the same fixed scratch array inside the library.  Collected last on purpose
so that a failure here cannot hide the results of the other tests."""

import ctypes

import numpy as np
import pytest

import oracle as O
import workload as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def setup():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_16915_gb300 import build
    build.build()
    import paper_2609_16915_gb300 as R
    from tests import gpu_util as G
    p = W.CONFIGS["standard"]
    bsk, ksk = W.uniform_keys(p, seed=21)
    ctx = G.make_ctx(p, bsk, ksk)
    return R, G, p, ctx


def _call_noalloc(R, ctx, lwe, lut, out):
    """Straight through the C ABI."""
    return R.load().rosetta_pbs_batch_noalloc(ctx._h, ctypes.c_void_p(lwe.data_ptr()), lwe.shape[0],
                                              ctypes.c_void_p(lut.data_ptr()), ctypes.c_void_p(out.data_ptr()),
                                              ctypes.c_void_p(None))


def test_noalloc_matches_pbs_batch_twice_in_a_row(setup):
    R, G, p, ctx = setup
    lut_h = W.lut_torus(p)
    lut = G.to_dev(lut_h)
    first_h = W.uniform_ciphertexts(p, 300, sub=31)
    first_h[[0, 299]] = G.sparse_lwe(p, 2, 3, seed=33)          # short chains at the ends
    first = G.to_dev(first_h)
    second = G.to_dev(W.uniform_ciphertexts(p, 77, sub=32))   # smaller: stale words from call 1 remain
    for call, lwe in enumerate((first, second)):
        want = G.empty_dev(lwe.shape[0], p.n + 1)
        ctx.pbs_batch(lwe, lut, want, stream=0)
        ctx.sync_status(stream=0)
        got = G.empty_dev(lwe.shape[0], p.n + 1)
        assert _call_noalloc(R, ctx, lwe, lut, got) == 0
        ctx.sync_status(stream=0)
        got_h = G.to_host(got)
        assert np.array_equal(got_h, G.to_host(want))
        if call == 0:
            # and against the CPU oracle at sampled positions (150: a dense
            # chain of all n CMux steps)
            pos = np.array([0, 150, 299])
            bsk, ksk = W.uniform_keys(p, seed=21)
            assert np.array_equal(got_h[pos], O.pbs_batch(p, bsk, ksk, first_h[pos], lut_h))


def test_noalloc_rejects_oversize_and_host_buffers(setup):
    R, G, p, ctx = setup
    lut = G.to_dev(W.lut_torus(p))
    limit = (2 << 20) // (p.kN + 1)                              # 16 MiB of 64-bit words
    big = G.to_dev(np.zeros((limit + 1, p.n + 1), np.uint64))
    out = G.empty_dev(limit + 1, p.n + 1)
    assert _call_noalloc(R, ctx, big, lut, out) == -1
    host_in = np.zeros((4, p.n + 1), np.uint64)
    st = R.load().rosetta_pbs_batch_noalloc(ctx._h, ctypes.c_void_p(host_in.ctypes.data), 4,
                                            ctypes.c_void_p(lut.data_ptr()), ctypes.c_void_p(out.data_ptr()),
                                            ctypes.c_void_p(None))
    assert st == -1
    ok_in = big[:limit]
    assert _call_noalloc(R, ctx, ok_in, lut, out[:limit]) == 0
    ctx.sync_status(stream=0)
    # a context's max_batch binds this entry point as it binds rosetta_pbs_batch
    bsk, ksk = W.uniform_keys(p, seed=21)
    small = G.make_ctx(p, bsk, ksk, max_batch=2)
    assert _call_noalloc(R, small, big[:3], lut, out[:3]) == -1
    assert _call_noalloc(R, small, big[:2], lut, out[:2]) == 0
    small.sync_status(stream=0)
    small.close()


def test_noalloc_on_a_three_prime_context(setup):
    """The N = 4096 set runs the three-prime kernel: the same words as
    rosetta_pbs_batch and, at a dense and a sparse position, as the oracle."""
    R, G, _, _ = setup
    p = W.CONFIGS["gpt2_mlp"]
    bsk, ksk = W.uniform_keys(p, seed=23)
    ctx = G.make_ctx(p, bsk, ksk)
    assert ctx.ntt_primes() == 3
    lut_h = W.lut_torus(p)
    lut = G.to_dev(lut_h)
    lwe_h = W.uniform_ciphertexts(p, 40, sub=34)
    lwe_h[[39]] = G.sparse_lwe(p, 1, 5, seed=35)
    lwe = G.to_dev(lwe_h)
    want = G.empty_dev(40, p.n + 1)
    ctx.pbs_batch(lwe, lut, want, stream=0)
    ctx.sync_status(stream=0)
    got = G.empty_dev(40, p.n + 1)
    assert _call_noalloc(R, ctx, lwe, lut, got) == 0
    ctx.sync_status(stream=0)
    got_h = G.to_host(got)
    assert np.array_equal(got_h, G.to_host(want))
    pos = np.array([7, 39])
    assert np.array_equal(got_h[pos], O.pbs_batch(p, bsk, ksk, lwe_h[pos], lut_h))
    ctx.close()
