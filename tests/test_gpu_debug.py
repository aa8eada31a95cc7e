"""The ROSETTA_DEBUG build (device-side bounds checks that report
ROSETTA_ERR_BOUNDS and skip the access, in place of a memory checker): it
computes the same words as the oracle, and a check made to fail on purpose
is reported once by rosetta_sync_status while the context stays usable.  The
regular build has no checks and says so."""

import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _libs():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_16915_gb300 import build
    build.build()
    build.build(debug=True)


def test_debug_build_bitexact_and_reports_bounds():
    r = subprocess.run([sys.executable, "-m", "tests.debug_client"], cwd=ROOT, capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0, r.stderr[-3000:]
    res = json.loads(r.stdout.strip().splitlines()[-1])
    assert res == {"tiny_bitexact": True, "standard_bitexact": True, "three_prime_bitexact": True, "bounds_status": -7,
                   "three_prime_bounds_status": -7, "after_bitexact": True}


def test_regular_build_has_no_bounds_checks():
    import paper_2609_16915_gb300 as R
    import workload as W
    from tests import gpu_util as G
    p = W.CONFIGS["tiny"]
    bsk, ksk = W.uniform_keys(p, seed=64)
    ctx = G.make_ctx(p, bsk, ksk)
    with pytest.raises(R.RosettaError) as e:
        ctx.selftest_bounds()
    assert e.value.status == -2
