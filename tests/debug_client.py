"""Run in a child process by tests/test_gpu_debug.py: load the library built
with -DROSETTA_DEBUG (a process holds one librosetta), bootstrap small
batches through it and compare with the CPU oracle, then make its bounds
check fail on purpose and check the report.  Prints one JSON line."""

import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import oracle as O  # noqa: E402
import paper_2609_16915_gb300 as R  # noqa: E402
import workload as W  # noqa: E402


def main():
    R.load(R.DEBUG_LIB_PATH)
    from tests import gpu_util as G
    res = {}
    p = W.CONFIGS["tiny"]
    keys = O.Keys(p, W.key_draws(p))
    lwe = keys.encrypt(W.cipher_draws(p, 37, sub=61))
    lut = W.lut_torus(p)
    ctx = G.make_ctx(p, keys.bsk, keys.ksk)
    res["tiny_bitexact"] = bool(np.array_equal(G.gpu_pbs(ctx, p, lwe, lut), O.pbs_batch(p, keys.bsk, keys.ksk, lwe, lut)))
    ps = W.CONFIGS["standard"]
    bsk, ksk = W.uniform_keys(ps, seed=62)
    sl = G.sparse_lwe(ps, 3, 4, seed=63)
    cs = G.make_ctx(ps, bsk, ksk)
    res["standard_bitexact"] = bool(np.array_equal(G.gpu_pbs(cs, ps, sl, W.lut_torus(ps)),
                                                   O.pbs_batch(ps, bsk, ksk, sl, W.lut_torus(ps))))
    ctx.selftest_bounds()
    try:
        ctx.sync_status()
        res["bounds_status"] = 0
    except R.RosettaError as e:
        res["bounds_status"] = e.status
    # reported once; the context keeps working
    res["after_bitexact"] = bool(np.array_equal(G.gpu_pbs(ctx, p, lwe, lut), O.pbs_batch(p, keys.bsk, keys.ksk, lwe, lut)))
    print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
