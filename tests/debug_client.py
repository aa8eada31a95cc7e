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
    # the three-prime kernel (N = 4096 set) under the same checks
    pg = W.CONFIGS["gpt2_mlp"]
    bg, kg = W.uniform_keys(pg, seed=65)
    gl = G.sparse_lwe(pg, 2, 3, seed=66)
    cg = G.make_ctx(pg, bg, kg)
    res["three_prime_bitexact"] = bool(cg.ntt_primes() == 3 and np.array_equal(
        G.gpu_pbs(cg, pg, gl, W.lut_torus(pg)), O.pbs_batch(pg, bg, kg, gl, W.lut_torus(pg))))
    for name, c in (("bounds_status", ctx), ("three_prime_bounds_status", cg)):
        c.selftest_bounds()
        try:
            c.sync_status()
            res[name] = 0
        except R.RosettaError as e:
            res[name] = e.status
    # reported once; the context keeps working
    res["after_bitexact"] = bool(np.array_equal(G.gpu_pbs(ctx, p, lwe, lut), O.pbs_batch(p, keys.bsk, keys.ksk, lwe, lut)))
    print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
