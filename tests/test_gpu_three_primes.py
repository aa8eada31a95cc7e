"""The three-prime blind rotation (primes just under 2^31, clusters of three
CTAs) against the oracle, and the rule that picks it.

A context takes three primes where the external product's bound
(k+1) l N 2^(beta-1) 2^63 stays within 0.45 of their product, the kernel
exists (16-bit digits, N = 4096 or 8192, l <= 3) and as many of its CTAs
fit one SM's shared memory as of the four-prime kernel's;
four primes otherwise.  The outputs are the same words either way, so every
case is compared word for word with the oracle: each compiled ring size and
level, the encrypted-test-polynomial variant, many LUTs, the largest
magnitude the rule admits at each ring size, and the four-prime kernels the
rule now bypasses at N = 4096."""

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


def _params(N, base_log, level, n, batch=3):
    return W.Params(f"t{N}_{base_log}x{level}_{n}", n=n, k=1, N=N, pbs_base_log=base_log, pbs_level=level,
                    ks_base_log=4, ks_level=4, msg_bits=3, lwe_sigma_log2=40, glwe_sigma_log2=20,
                    lut=("square_mod",), msg=("uniform",), batch=batch, seed=N + 7 * base_log + level + n)


def _br3_smem(N, level, n):
    """Shared memory of one three-prime CTA (the kernel's layout: twiddles,
    owned accumulator words, the exchange buffer extended to 12 T words for
    the outgoing residues, packed digits, the switched mask)."""
    T = N // 8
    b = 8 * N + 48 * T + 4 * (12 * T + 3 * level * T) + 2 * (n + 1)
    return (b + 15) & ~15


def _br4_smem(N, level, n):
    """Shared memory of one four-prime CTA with 16-bit digits (N >= 2048):
    twiddles, accumulator quarter, the exchange buffer of 2N words that also
    holds the outgoing residues, digits, the switched mask."""
    Q = N // 4
    b = 8 * N + 16 * Q + 8 * N + 4 * level * Q + 2 * (n + 1)
    return (b + 15) & ~15


def _primes(p):
    import paper_2609_16915_gb300 as R
    ctx = R.Context(p, device=0)
    try:
        return ctx.ntt_primes()
    finally:
        ctx.close()


@pytest.mark.parametrize("name,want", [("gpt2_mlp", 3), ("llama_silu", 3), ("standard", 4), ("paper_dims", 4),
                                       ("tiny", 4)])
def test_named_sets_take_the_expected_prime_set(name, want):
    """N = 4096 (l = 2, beta = 15: bound 0.25 of the three primes' product)
    and N = 8192 (l = 3, beta = 14: 0.375) take three; N = 2048 with
    beta = 23 needs four (bound above 2^97); N = 256 has no three-prime
    kernel."""
    assert _primes(W.CONFIGS[name]) == want


def test_rule_at_the_bound_and_at_the_shared_memory_limit():
    import torch
    # beta = 16, l = 2 at N = 4096: bound 0.50 of the product, over 0.45
    assert _primes(_params(4096, 16, 2, 3)) == 4
    assert _primes(_params(4096, 15, 3, 3)) == 3                  # 0.375
    # three primes only while their CTAs fit an SM as densely as the four-prime
    # kernel's (1 KB reserved per CTA): the rule at every n up to 12000, and
    # the context's choice at the ends and around every change
    props = torch.cuda.get_device_properties(0)
    per_sm = getattr(props, "shared_memory_per_multiprocessor", None)
    if per_sm is None:
        pytest.skip("this torch does not report shared memory per SM")
    fits = lambda b: per_sm // (b + 1024)
    for N, beta, level in ((4096, 15, 2), (8192, 14, 3)):
        top = 14000 if N == 4096 else 22015                       # beyond: the four-prime kernel's own limit
        rule = [fits(_br3_smem(N, level, n)) >= fits(_br4_smem(N, level, n)) for n in range(1, top + 1)]
        flips = [n for n in range(2, top + 1) if rule[n - 1] != rule[n - 2]]
        for n in sorted({1, top} | {m for f in flips for m in (f - 1, f)}):
            assert _primes(_params(N, beta, level, n)) == (3 if rule[n - 1] else 4), (N, n)


@pytest.mark.parametrize("N,base_log,level", [(4096, 16, 1), (4096, 12, 1), (4096, 15, 2), (4096, 12, 2),
                                              (4096, 15, 3), (4096, 11, 3),
                                              (8192, 15, 1), (8192, 14, 2), (8192, 14, 3), (8192, 11, 3)])
def test_every_three_prime_level_bitexact(N, base_log, level):
    """Dense masks on a short LWE (every CMux step runs), every output word
    of blind rotation + extraction and of the whole PBS."""
    p = _params(N, base_log, level, 4 if N == 4096 else 2, batch=3 if N == 4096 else 2)
    bsk, ksk = W.uniform_keys(p)
    lwe = W.uniform_ciphertexts(p, p.batch, sub=3)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, bsk, ksk)
    assert ctx.ntt_primes() == 3
    big = G.gpu_br_extract(ctx, p, lwe, lut)
    want = O.blind_rotate_extract_batch(p, bsk, lwe, lut)
    assert np.array_equal(big, want)
    assert np.array_equal(G.gpu_pbs(ctx, p, lwe, lut), O.keyswitch_batch(p, ksk, want))
    ctx.close()


@pytest.mark.parametrize("N,base_log,level", [(4096, 15, 2), (8192, 14, 3)])
def test_three_prime_glwe_test_polynomials_and_many_luts(N, base_log, level):
    """The per-ciphertext GLWE test polynomial variant and per-ciphertext
    LUT selection on the three-prime kernel."""
    p = _params(N, base_log, level, 3 if N == 4096 else 2, batch=4)
    bsk, ksk = W.uniform_keys(p)
    lwe = W.uniform_ciphertexts(p, p.batch, sub=5)
    g = np.random.default_rng(77)
    glwe = g.integers(0, 2**64, size=(p.batch, p.k + 1, p.N), dtype=np.uint64, endpoint=False)
    ctx = G.make_ctx(p, bsk, ksk)
    assert ctx.ntt_primes() == 3
    out = G.empty_dev(p.batch, p.k + 1, p.N)
    ctx.blind_rotate_glwe_batch(G.to_dev(lwe), G.to_dev(glwe), out)
    ctx.sync_status()
    assert np.array_equal(G.to_host(out), O.blind_rotate_glwe_batch(p, bsk, lwe, glwe))
    luts = np.stack([W.lut_torus(p, codes=[(m * (j + 1) + j) % 8 for m in range(8)]) for j in range(3)])
    import torch
    idx = np.array([2, 0, 1, 2])
    got = G.empty_dev(p.batch, p.n + 1)
    ctx.pbs_batch_multi_lut(G.to_dev(lwe), G.to_dev(luts), torch.from_numpy(idx.astype(np.int32)).cuda(), got)
    ctx.sync_status()
    assert np.array_equal(G.to_host(got), O.pbs_batch_multi_lut(p, bsk, ksk, lwe, luts, idx))
    ctx.close()


@pytest.mark.parametrize("N,base_log,level,share", [(4096, 15, 3, 0.374), (8192, 14, 3, 0.374)])
@pytest.mark.parametrize("sign", [+1, -1])
def test_three_prime_product_at_the_largest_admitted_magnitude(N, base_log, level, share, sign):
    """Every digit at -B/2 against key words of one sign close to 2^63, so
    coefficient N-1 sums 2 l N terms of one sign: 3 x 2^90 = 0.375 of the
    three primes' product with l = 3, beta = 15 at N = 4096, 3 x 2^91 = 0.375
    with l = 3, beta = 14 at N = 8192 (the largest bounds among the sets
    that take three primes at these ring sizes).  Against the oracle and the
    closed form."""
    p = _params(N, base_log, level, 2, batch=1)
    bsk, lwe, glwe, C = X.case(p, sign, seed=41)
    ksk = W.uniform_keys(p)[1]
    ctx = G.make_ctx(p, bsk, ksk)
    assert ctx.ntt_primes() == 3
    out = G.empty_dev(1, p.k + 1, p.N)
    ctx.blind_rotate_glwe_batch(G.to_dev(lwe), G.to_dev(glwe), out)
    ctx.sync_status()
    got = G.to_host(out)
    assert np.array_equal(got, O.blind_rotate_glwe_batch(p, bsk, lwe, glwe))
    want, peak = X.expected(p, bsk, C)
    assert peak > share * 2**92.999
    assert [[int(w) for w in row] for row in got[0]] == want
    ctx.close()


@pytest.mark.parametrize("base_log,level,n", [(16, 2, 4), (16, 3, 4), (16, 2, 5000)])
def test_four_prime_kernels_the_rule_bypasses(base_log, level, n):
    """The four-prime kernels with 16-bit digits at N = 4096 that the
    three-prime rule leaves to sets whose bound exceeds 0.45 of the three
    primes' product: two and three levels with beta = 16 (bounds 0.50 and
    0.75), also at n = 5000 (one CTA per SM; sparse masks, 12 CMux steps, one
    at the last index).  With one level and beta <= 16 the bound is at most
    0.25 and the CTA no larger than the four-prime one: every such set takes
    three primes."""
    p = _params(4096, base_log, level, n, batch=2)
    bsk, ksk = W.uniform_keys(p)
    if n > 100:
        lwe = G.sparse_lwe(p, p.batch, 12, seed=level)
        lwe[:, p.n - 1] = np.uint64(3 << 60)
    else:
        lwe = W.uniform_ciphertexts(p, p.batch, sub=9)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, bsk, ksk)
    assert ctx.ntt_primes() == 4
    assert np.array_equal(G.gpu_br_extract(ctx, p, lwe, lut), O.blind_rotate_extract_batch(p, bsk, lwe, lut))
    ctx.close()


def test_three_prime_bad_lut_index_is_reported_not_followed():
    """An out-of-range LUT index on the three-prime kernel: that ciphertext
    takes LUT 0, the others their own, and the next rosetta_sync_status
    reports INVALID_ARG once."""
    import torch
    import paper_2609_16915_gb300 as R
    p = _params(4096, 15, 2, 3, batch=3)
    bsk, ksk = W.uniform_keys(p)
    lwe = W.uniform_ciphertexts(p, p.batch, sub=8)
    luts = np.stack([W.lut_torus(p), W.lut_torus(p, codes=[(5 * m + 1) % 8 for m in range(8)])])
    idx = np.array([1, 7, 0])
    ctx = G.make_ctx(p, bsk, ksk)
    assert ctx.ntt_primes() == 3
    out = G.empty_dev(p.batch, p.n + 1)
    ctx.pbs_batch_multi_lut(G.to_dev(lwe), G.to_dev(luts), torch.from_numpy(idx.astype(np.int32)).cuda(), out)
    with pytest.raises(R.RosettaError) as e:
        ctx.sync_status()
    assert e.value.status == -1
    ctx.sync_status()                                    # reported once
    assert np.array_equal(G.to_host(out), O.pbs_batch_multi_lut(p, bsk, ksk, lwe, luts, np.array([1, 0, 0])))
    ctx.close()
