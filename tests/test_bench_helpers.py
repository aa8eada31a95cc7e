"""Host-side helpers of bench.py: operation counts, the key-switch path the
library takes, the traffic summary lookup.  CPU only."""

import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import workload as W  # noqa: E402


def test_operation_counts_of_the_standard_set():
    """4 primes at N = 2048 (98 bits needed), 1.37 G integer ops of blind rotation per PBS."""
    p = W.CONFIGS["standard"]
    assert bench.min_primes(p) == 4
    br, ks = bench.int_ops_per_pbs(p)
    assert br == pytest.approx(1.368e9, rel=2e-3)
    assert ks == p.kN * p.ks_level * (p.n + 1) * 3 + p.kN * p.ks_level * 6


def test_counting_convention_uses_three_primes_for_the_large_rings():
    for name in ("gpt2_mlp", "llama_silu"):
        assert bench.min_primes(W.CONFIGS[name]) == 3


def test_key_switch_path_selection():
    """Mirrors the library's rule: tensor cores from 256 ciphertexts on, 8
    limbs when 2^(beta-1) 255 K < 2^24, else 16 when 2^(beta-1) 15 K < 2^24."""
    assert bench.ks_tensor_limbs(W.CONFIGS["standard"], 4096) == 8
    assert bench.ks_tensor_limbs(W.CONFIGS["standard"], 255) == 0
    assert bench.ks_tensor_limbs(W.CONFIGS["gpt2_mlp"], 3072) == 16
    assert bench.ks_tensor_limbs(W.CONFIGS["llama_silu"], 14336) == 16
    assert bench.ks_tensor_flops(W.CONFIGS["standard"], 4096, 8) == 2.0 * 4096 * 10240 * 6144


def test_traffic_summary_only_for_its_own_workload():
    assert bench.measured_traffic(W.CONFIGS["gpt2_mlp"], 3072) is None
    assert bench.measured_traffic(W.CONFIGS["standard"], 1024) is None


def test_lookup_operation_counts_are_dominated_by_blind_rotation():
    ops = bench.int_ops_per_lookup(W.CONFIGS["standard"], 4, 16, 4)
    assert ops["blind_rotation"] == 6 * bench.int_ops_per_pbs(W.CONFIGS["standard"])[0]
    assert ops["blind_rotation"] / sum(ops.values()) > 0.97
