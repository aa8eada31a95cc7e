"""Key switch parity on both kernels: the tensor-core one (batches of 256 and
more, where its fp32 sums are exact) and the split-K CUDA-core one.  Every
output word is compared with the oracle."""

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


@pytest.mark.parametrize("name,batch", [("standard", 300), ("standard", 256), ("gpt2_mlp", 260),
                                        ("llama_silu", 257), ("tiny", 385), ("standard", 100)])
def test_keyswitch_bitexact(name, batch):
    """Uniform-word keys and inputs; ragged last tile of 128 ciphertexts."""
    p = W.CONFIGS[name]
    _, ksk = W.uniform_keys(p, seed=91)
    big = W.uniform_u64((batch, p.kN + 1), W.rng(p.seed, "sample", 95))
    import paper_2609_16915_gb300 as R
    ctx = R.Context(p)
    ctx.upload_ksk(G.to_dev(ksk))
    assert np.array_equal(G.gpu_keyswitch(ctx, p, big), O.keyswitch_batch(p, ksk, big))


def test_keyswitch_extreme_digits():
    """Every digit at -B/2 and every key word 2^64 - 1: the largest partial
    sums the tensor-core path can see."""
    p = W.CONFIGS["standard"]
    ksk = np.full(p.ksk_shape(), np.uint64(2**64 - 1), np.uint64)
    # a' whose rounded value makes every balanced digit -B/2: v + C = 0 mod 2^(beta l)
    bits = p.ks_base_log * p.ks_level
    B = 1 << p.ks_base_log
    C = sum((B >> 1) << (m * p.ks_base_log) for m in range(p.ks_level))
    v = (-C) % (1 << bits)
    a = (v << (64 - bits)) % (1 << 64)
    big = np.full((300, p.kN + 1), np.uint64(a), np.uint64)
    import paper_2609_16915_gb300 as R
    ctx = R.Context(p)
    ctx.upload_ksk(G.to_dev(ksk))
    assert np.array_equal(G.gpu_keyswitch(ctx, p, big), O.keyswitch_batch(p, ksk, big))


def test_expired_wait_is_reported_and_the_context_stays_usable():
    """A bounded wait that nothing completes gives up, sync_status reports
    TIMEOUT once, and the next key switch on the same context is exact."""
    import paper_2609_16915_gb300 as R
    p = W.CONFIGS["standard"]
    _, ksk = W.uniform_keys(p, seed=93)
    ctx = R.Context(p)
    ctx.upload_ksk(G.to_dev(ksk))
    ctx.sync_status()
    ctx.selftest_wait_timeout(20000)
    with pytest.raises(R.RosettaError) as e:
        ctx.sync_status()
    assert e.value.status == -6
    ctx.sync_status()                                # reported once, then cleared
    big = W.uniform_u64((300, p.kN + 1), W.rng(p.seed, "sample", 97))
    assert np.array_equal(G.gpu_keyswitch(ctx, p, big), O.keyswitch_batch(p, ksk, big))
