"""The seeded inputs are the same on every host: the workload module's draws
for every parameter set hash to the values in tests/golden/input_manifest.json
(written by tests/golden/make_input_manifest.py from the workload module
alone).  The draws use only the raw PCG64 stream, which numpy keeps fixed
across versions; this test catches any change that would alter them."""

import json
import os

import numpy as np
import pytest

import workload as W
from tests.golden.make_input_manifest import OUT, digests

MAN = json.load(open(OUT))


@pytest.mark.parametrize("name", sorted(MAN["sha256"]))
def test_draws_match_manifest(name):
    assert W.CONFIGS[name].batch == MAN["batch"][name]
    assert digests(name) == MAN["sha256"][name]


def test_normal_variates_moments():
    """The Irwin-Hall variates have mean 0 and variance 1 (1e6 samples), and
    the rounding of gaussian_u64 is exact integer arithmetic."""
    g = W.rng(123, "sample")
    z = W.standard_normal(1_000_000, g)
    assert abs(z.mean()) < 5e-3 and abs(z.var() - 1.0) < 5e-3 and np.abs(z).max() < 6.0
    g1, g2 = W.rng(9, "sample", 1), W.rng(9, "sample", 1)
    zf = W.normal_fixed(1000, g1)
    v = W.gaussian_u64((1000,), 20, g2).view(np.int64)
    want = np.array([(int(x) + (1 << 32)) >> 33 for x in zf], np.int64)   # round half up of x / 2^33
    assert np.array_equal(v, want)


def test_manifest_names_every_config():
    assert set(MAN["sha256"]) == set(W.CONFIGS)
