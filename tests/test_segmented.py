"""Segmented-LUT builder and cleartext three-step lookup, pinned by the
paper's running example (1/x on [0.1, 2.0])."""

import json
import os

import numpy as np
import pytest

from paper_2609_16915_gb300 import segmented as SG
import workload as W

G = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_segmented_example.json")))
INV = SG.FUNCTIONS["reciprocal"]


def _grid(lo, hi, n=200001):
    return np.linspace(lo, hi, n, endpoint=False)


@pytest.fixture(scope="module")
def lut():
    return SG.build(INV, G["tau"], G["n_br"])


def test_indices_and_value_at_the_example_point(lut):
    x = G["x"]
    assert SG.segment_index(lut, x) == G["segment"]
    assert SG.interval_index(lut, x, G["segment"]) == G["interval"]
    assert lut.a[0, 1] == pytest.approx(G["a01"], abs=5e-4)
    assert lut.b[0, 1] == pytest.approx(G["b01"], abs=5e-4)
    assert SG.lookup(lut, x) == pytest.approx(G["value"], abs=5e-4)
    assert abs(SG.lookup(lut, x) - 1 / x) / (1 / x) == pytest.approx(G["relative_error_linear_at_x"], abs=5e-4)


def test_printed_slope_and_offset_polynomials(lut):
    a0, b0 = SG.value_polynomials(lut, 0)
    assert np.allclose(a0, G["a0_coeffs"], atol=5e-3)
    assert np.allclose(b0, G["b0_coeffs"], atol=5e-3)
    p, q = SG.index_polynomials(lut)
    assert np.allclose(p, G["p_coeffs"], atol=5e-4)
    assert np.allclose(q, G["q_coeffs"], atol=5e-4)
    # t = p x + q: each segment's candidate interval position
    assert np.allclose(p * G["x"] + q, G["t"], atol=5e-4)


def test_candidate_values_of_both_segments(lut):
    for s, key in [(0, "r0"), (1, "r1")]:
        a, b = SG.value_polynomials(lut, s)
        assert np.allclose(a * G["x"] + b, G[key], atol=2.5e-3)


def test_error_figures_of_the_running_example(lut):
    lo, hi = G["tau"][0], G["tau"][-1]
    xs = _grid(lo, hi)
    # single staircase LUT of N_br midpoints (the one-PBS baseline)
    mids = W.bin_midpoints(lo, hi, G["n_br"])
    stair = np.array([1 / mids[W.bin_index(x, lo, hi, G["n_br"])] for x in xs])
    rel = np.abs(stair - 1 / xs) * xs
    assert rel.max() == pytest.approx(G["max_relative_error_single_lut"], abs=1e-3)
    x = G["x"]
    assert abs(1 / mids[0] - 1 / x) * x == pytest.approx(G["relative_error_baseline_at_x"], abs=1e-3)
    # two segments, constant (midpoint) entries
    const = []
    for v in xs:
        s = SG.segment_index(lut, v)
        i = SG.interval_index(lut, v, s)
        w = (lut.tau[s + 1] - lut.tau[s]) / lut.n_br
        const.append(1 / (lut.tau[s] + (i + 0.5) * w))
    assert (np.abs(np.array(const) - 1 / xs) * xs).max() == pytest.approx(
        G["max_relative_error_two_segments_constant"], abs=1e-3)
    # two segments, linear entries
    lin = np.array([SG.lookup(lut, v) for v in xs[::10]])
    assert (np.abs(lin - 1 / xs[::10]) * xs[::10]).max() == pytest.approx(
        G["max_relative_error_two_segments_linear"], abs=1.5e-3)


def test_boundaries():
    t = SG.boundaries(0.1, 2.0, 4, "log")
    assert t[0] == pytest.approx(0.1) and t[-1] == pytest.approx(2.0)
    assert np.allclose(np.diff(np.log(t)), np.log(20) / 4)
    u = SG.boundaries(-4, 4, 4, "uniform")
    assert u == [-4, -2, 0, 2, 4]
    with pytest.raises(ValueError):
        SG.boundaries(0.0, 2.0, 4, "log")


@pytest.mark.parametrize("name,lo,hi,spacing", [("gelu", -20, 20, "uniform"), ("silu", -20, 20, "uniform"),
                                                ("reciprocal", 0.1, 100, "log"), ("rsqrt", 0.1, 100, "log")])
def test_linear_segments_beat_the_staircase(name, lo, hi, spacing):
    """With N_seg = 4 segments (the paper's setting) the linear tables are far
    more accurate than one staircase LUT of the same N_br."""
    f = SG.FUNCTIONS[name]
    n_br = 64
    lut = SG.build(f, SG.boundaries(lo, hi, 4, spacing), n_br)
    xs = _grid(lo, hi, 20001)
    exact = np.array([f(v) for v in xs])
    seg = np.array([SG.lookup(lut, v) for v in xs])
    mids = W.bin_midpoints(lo, hi, n_br)
    stair = np.array([f(mids[W.bin_index(v, lo, hi, n_br)]) for v in xs])
    assert np.sqrt(np.mean((seg - exact) ** 2)) < 0.2 * np.sqrt(np.mean((stair - exact) ** 2))
