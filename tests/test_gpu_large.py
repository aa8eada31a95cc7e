"""Parity of the two large parameter sets (N = 4096: gpt2_mlp, N = 8192:
llama_silu) over whole launches and long dense CMux chains.

These sets run their own kernel specialisations (two and three gadget
levels, 16-bit digits, named-barrier groups, one or two CTAs per SM), so a
race or a barrier slip that needs full occupancy or many steps to show must
be looked for at their full batch sizes:

* every output of the full launch (3072 and 14336 dense ciphertexts, so
  nearly every one of the n CMux steps runs) against the closed form of PBS
  under noiseless keys (tests/closed_form.py);
* real keys over the full launch: two positions carry long dense chains
  (all 840 steps at N = 4096, 64 at N = 8192) compared word for word with the
  CPU oracle, and every other output decrypts to the LUT.
"""

import numpy as np
import pytest

import oracle as O
import workload as W
from tests import closed_form as CF
from tests import gpu_util as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_16915_gb300 import build
    build.build()


def _bijective_lut(p):
    """A LUT whose codes are all distinct, so a wrong box index cannot land
    on an equal entry."""
    return W.lut_torus(p, codes=[(37 * m + 11) % (1 << p.msg_bits) for m in range(1 << p.msg_bits)])


@pytest.mark.parametrize("name", ["gpt2_mlp", "llama_silu"])
def test_full_batch_noiseless_keys_every_output(name):
    p = W.CONFIGS[name]
    d = W.key_draws(p, trivial=True)
    bsk = CF.noiseless_bsk(p, d.lwe_key)
    ksk = CF.noiseless_ksk(p, d.glwe_key)
    lut = _bijective_lut(p)
    lwe = W.uniform_ciphertexts(p, p.batch, sub=41)
    ctx = G.make_ctx(p, bsk, ksk, max_batch=p.batch)
    got = G.gpu_pbs(ctx, p, lwe, lut)
    ctx.close()
    steps = int(np.count_nonzero(CF.modswitch(lwe[:, :p.n], p.N)))
    assert steps > 0.99 * p.batch * p.n                  # the chains are dense
    assert not got[:, :p.n].any()
    body = CF.noiseless_pbs_body(p, d.lwe_key, lwe, lut)
    bad = np.flatnonzero(got[:, p.n] != body)
    assert bad.size == 0, f"{bad.size} of {p.batch} bodies differ, first at {bad[:8]}"


@pytest.mark.parametrize("name,dense,pos_sub", [("gpt2_mlp", None, 6), ("llama_silu", 64, 7)])
def test_full_batch_real_keys_dense_chains_and_decrypt(name, dense, pos_sub):
    """dense=None: the two checked positions are uniform words (every step
    runs); otherwise they have `dense` nonzero mask words."""
    p = W.CONFIGS[name]
    keys = O.Keys(p, W.key_draws(p))
    cd = W.cipher_draws(p, p.batch, sub=pos_sub)
    lwe = keys.encrypt(cd)
    pos = np.array([1, p.batch - 2])
    if dense is None:
        lwe[pos] = W.uniform_ciphertexts(p, len(pos), sub=50 + pos_sub)
    else:
        lwe[pos] = G.sparse_lwe(p, len(pos), dense, seed=50 + pos_sub)
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk, max_batch=p.batch)
    got = G.gpu_pbs(ctx, p, lwe, lut)
    ctx.close()
    assert np.array_equal(got[pos], O.pbs_batch(p, keys.bsk, keys.ksk, lwe[pos], lut))
    others = np.setdiff1d(np.arange(p.batch), pos)
    fails = int(np.sum(keys.decrypt(got[others]) != W.lut_codes(p)[cd.codes[others]]))
    assert fails == 0
