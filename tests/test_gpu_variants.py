"""Every compiled blind-rotation specialisation against the oracle.

The blind-rotation kernel is specialised on the ring size, the digit width
(16-bit digits when the gadget base is at most 2^16) and, from N = 2048 up,
the gadget level count (1, 2, 3, or any).  At N = 4096 and 8192 the
16-bit-digit cases whose product bound is small enough run the three-prime
kernel (the context picks it where the bound allows; (8192, 15, 2),
(8192, 16, 1) and (8192, 16, 3) stay on four primes, and
tests/test_gpu_three_primes.py reaches the four-prime kernels at N = 4096).  Each case picks a gadget that
lands on one specialisation the headline parameter sets do not reach; dense
masks on a short LWE keep the oracle's schoolbook products quick.  Parameter
sets whose CTA does not fit the shared memory of one SM are refused at
context creation.  The last test drives the exact external product to the
largest magnitude the accepted parameters allow."""

import numpy as np
import pytest

import oracle as O
import workload as W
from tests import extreme_util as X
from tests import gpu_util as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_16915_gb300 import build
    build.build()


def _params(N, base_log, level, n):
    return W.Params(f"v{N}_{base_log}x{level}", n=n, k=1, N=N, pbs_base_log=base_log, pbs_level=level,
                    ks_base_log=4, ks_level=4, msg_bits=3, lwe_sigma_log2=40, glwe_sigma_log2=20,
                    lut=("square_mod",), msg=("uniform",), batch=2, seed=N + 7 * base_log + level)


# (N, beta, l): 16-bit digits for beta <= 16, else 32-bit; l >= 4 takes the
# run-time level loop.  beta * l = 64 (N = 2048, 16 x 4) is the gadget that
# reaches the last bit of the torus.
VARIANTS = [
    (256, 24, 2), (512, 28, 1), (1024, 8, 6),
    (2048, 16, 1), (2048, 13, 2), (2048, 11, 3), (2048, 16, 4), (2048, 28, 1), (2048, 24, 2), (2048, 21, 3),
    (4096, 16, 1), (4096, 12, 2), (4096, 11, 3), (4096, 9, 5), (4096, 28, 1), (4096, 24, 2), (4096, 21, 3),
    (8192, 16, 1), (8192, 10, 2), (8192, 15, 2), (8192, 16, 3), (8192, 28, 1),
    (8192, 12, 4), (8192, 20, 2), (8192, 17, 3),
]


@pytest.mark.parametrize("N,base_log,level", VARIANTS)
def test_every_specialisation_bitexact(N, base_log, level):
    n, count = (2, 1) if N == 8192 else (3, 2)
    p = _params(N, base_log, level, n)
    bsk, ksk = W.uniform_keys(p)
    lwe = W.uniform_ciphertexts(p, count, sub=1)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, bsk, ksk)
    got = G.gpu_br_extract(ctx, p, lwe, lut)
    assert np.array_equal(got, O.blind_rotate_extract_batch(p, bsk, lwe, lut))


@pytest.mark.parametrize("N,base_log,level,n", [(8192, 14, 3, 22016), (8192, 12, 4, 17920), (8192, 20, 2, 17920),
                                                 (8192, 17, 3, 9728)])
def test_parameter_sets_beyond_shared_memory_are_refused(N, base_log, level, n):
    """At N = 8192 the four-prime CTA (twiddles 64 KB, accumulator quarter
    32 KB, exchange buffer 64 KB) leaves 72 KB of the 227 KB a CTA may have
    for the digits (8 KB per level of 16-bit digits, 16 KB of 32-bit ones)
    and the a~_i (2 bytes each): the first n past the limit is refused, the
    one before it accepted."""
    import paper_2609_16915_gb300 as R
    with pytest.raises(R.RosettaError) as e:
        R.Context(_params(N, base_log, level, n), device=0)
    assert e.value.status == -2
    if n > 2:
        R.Context(_params(N, base_log, level, n - 1), device=0).close()


@pytest.mark.parametrize("N,base_log,level", [(2048, 28, 2), (4096, 28, 2), (8192, 28, 1)])
@pytest.mark.parametrize("sign", [+1, -1])
def test_external_product_at_its_largest_magnitude(N, base_log, level, sign):
    """Every digit at -B/2 against key words of one sign close to 2^63:
    coefficient N-1 sums (k+1) l N terms of one sign, about 2^104 here
    against the primes' product of about 2^112.  Checked against the oracle
    and, coefficient by coefficient, against the closed form."""
    p = _params(N, base_log, level, 2)
    bsk, lwe, glwe, C = X.case(p, sign, seed=N + level)
    ksk = W.uniform_keys(p)[1]
    ctx = G.make_ctx(p, bsk, ksk)
    out = G.empty_dev(1, p.k + 1, p.N)
    ctx.blind_rotate_glwe_batch(G.to_dev(lwe), G.to_dev(glwe), out)
    ctx.sync_status()
    got = G.to_host(out)
    assert np.array_equal(got, O.blind_rotate_glwe_batch(p, bsk, lwe, glwe))
    want, peak = X.expected(p, bsk, C)
    assert peak > 1 << 100
    assert [[int(w) for w in row] for row in got[0]] == want


@pytest.mark.parametrize("n", [1, 65535])
def test_lwe_dimension_extremes(n):
    """The smallest and the largest LWE dimension the library accepts (the
    a~_i are kept in shared memory as 16-bit words); nonzero masks at the
    first and the last index, so the first and the last CMux step both run."""
    p = W.Params(f"n{n}", n=n, k=1, N=256, pbs_base_log=16, pbs_level=1, ks_base_log=4, ks_level=4, msg_bits=3,
                 lwe_sigma_log2=40, glwe_sigma_log2=20, lut=("square_mod",), msg=("uniform",), batch=2, seed=n)
    bsk, ksk = W.uniform_keys(p)
    g = np.random.default_rng(n)
    lwe = np.zeros((2, n + 1), np.uint64)
    for b in range(2):
        for i in {0, n - 1, n // 2}:
            lwe[b, i] = g.integers(0, 2**64, dtype=np.uint64, endpoint=False)
        lwe[b, n] = g.integers(0, 2**64, dtype=np.uint64, endpoint=False)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, bsk, ksk)
    big = G.gpu_br_extract(ctx, p, lwe, lut)
    want_big = O.blind_rotate_extract_batch(p, bsk, lwe, lut)
    assert np.array_equal(big, want_big)
    assert np.array_equal(G.gpu_pbs(ctx, p, lwe, lut), O.keyswitch_batch(p, ksk, want_big))
    import paper_2609_16915_gb300 as R
    if n == 65535:
        with pytest.raises(R.RosettaError) as e:
            R.Context(W.Params(**{**p.__dict__, "n": 65536}), device=0)
        assert e.value.status == -2
