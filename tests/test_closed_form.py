"""CPU checks of the vectorised noiseless-key closed forms (tests/closed_form.py)
that the full-batch GPU tests compare against: they must agree with the
scalar closed form that pins the oracle, and the noiseless keys they build
from the GGSW / key-switching-key definitions must be the oracle's own keys
when its key generation is given zero masks and zero noise."""

import numpy as np
import pytest

import oracle as O
import workload as W
from tests import closed_form as CF
from tests.test_oracle import _closed_form_pbs


@pytest.mark.parametrize("name", ["tiny", "standard", "gpt2_mlp", "llama_silu"])
def test_vectorised_closed_form_matches_scalar(name):
    p = W.CONFIGS[name]
    s = W.key_draws(p, trivial=True).lwe_key
    lut = W.lut_torus(p, codes=[(37 * m + 11) % (1 << p.msg_bits) for m in range(1 << p.msg_bits)])
    lwe = W.uniform_ciphertexts(p, 24, sub=77)
    # the rounding edges of the modulus switch: a half step below/at/above, and words near 2^64
    sh = 64 - (2 * p.N).bit_length() + 1
    lwe[0, :] = np.uint64((1 << (sh - 1)) - 1)
    lwe[1, :] = np.uint64(1 << (sh - 1))
    lwe[2, :] = np.uint64(2**64 - 1)
    lwe[3, :] = np.uint64(2**64 - (1 << (sh - 1)))
    got = CF.noiseless_pbs_body(p, s, lwe, lut)
    want = np.array([_closed_form_pbs(p, s, lwe[b], lut) for b in range(lwe.shape[0])], np.uint64)
    assert np.array_equal(got, want)


def test_noiseless_keys_are_the_oracles_keys():
    for name in ["tiny", "lookup_small"]:
        p = W.CONFIGS[name]
        d = W.key_draws(p, trivial=True)
        keys = O.Keys(p, d)
        assert np.array_equal(CF.noiseless_bsk(p, d.lwe_key), keys.bsk)
        assert np.array_equal(CF.noiseless_ksk(p, d.glwe_key), keys.ksk)


@pytest.mark.parametrize("name", ["gpt2_mlp", "llama_silu"])
def test_noiseless_bsk_rows_at_full_size(name):
    """Two GGSWs of the large sets (one per key bit value) against the
    oracle's GGSW encryption with zero draws."""
    p = W.CONFIGS[name]
    d = W.key_draws(p, trivial=True)
    bsk = CF.noiseless_bsk(p, d.lwe_key)
    rows = (p.k + 1) * p.pbs_level
    zm = np.zeros((rows, p.k, p.N), np.uint64)
    zn = np.zeros((rows, p.N), np.uint64)
    for i in [int(np.argmin(d.lwe_key)), int(np.argmax(d.lwe_key))]:
        want = O.ggsw_encrypt(d.glwe_key, int(d.lwe_key[i]), p.pbs_base_log, p.pbs_level, zm, zn)
        assert np.array_equal(bsk[i], want)


def test_noiseless_oracle_pbs_matches_vectorised_closed_form():
    p = W.CONFIGS["tiny"]
    d = W.key_draws(p, trivial=True)
    lut = W.lut_torus(p, codes=[(5 * m + 3) % 8 for m in range(8)])
    lwe = W.uniform_ciphertexts(p, 32, sub=78)
    out = O.pbs_batch(p, CF.noiseless_bsk(p, d.lwe_key), CF.noiseless_ksk(p, d.glwe_key), lwe, lut)
    assert not out[:, :p.n].any()
    assert np.array_equal(out[:, p.n], CF.noiseless_pbs_body(p, d.lwe_key, lwe, lut))
