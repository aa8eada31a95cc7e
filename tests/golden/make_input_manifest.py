"""Write tests/golden/input_manifest.json: the SHA-256 of every seeded input
the workload module draws for each parameter set (keys' random draws, the
headline batch of ciphertext draws, the uniform-word keys and ciphertexts of
the timing runs, the LUT codes).  It calls only ``workload``: inputs, no
expected values.  tests/test_inputs.py regenerates the draws and compares,
so a host whose numpy produced other draws fails loudly instead of running
the real-key tests on different inputs.

    python tests/golden/make_input_manifest.py
"""

import hashlib
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))
import workload as W  # noqa: E402

OUT = os.path.join(HERE, "input_manifest.json")


def sha(a) -> str:
    a = np.ascontiguousarray(a)
    return hashlib.sha256(a.dtype.str.encode() + str(a.shape).encode() + a.tobytes()).hexdigest()


def digests(name: str) -> dict:
    p = W.CONFIGS[name]
    d = {}
    kd = W.key_draws(p)
    for f in ("lwe_key", "glwe_key", "bsk_mask", "bsk_noise", "ksk_mask", "ksk_noise"):
        d[f"key_draws.{f}"] = sha(getattr(kd, f))
    del kd
    cd = W.cipher_draws(p, p.batch)
    for f in ("codes", "mask", "noise"):
        d[f"cipher_draws.{f}"] = sha(getattr(cd, f))
    bsk, ksk = W.uniform_keys(p)
    d["uniform_keys.bsk"], d["uniform_keys.ksk"] = sha(bsk), sha(ksk)
    del bsk, ksk
    d["uniform_ciphertexts"] = sha(W.uniform_ciphertexts(p, p.batch))
    d["lut_codes"] = sha(W.lut_codes(p))
    return d


def main():
    man = {"numpy_at_write": np.__version__, "batch": {n: W.CONFIGS[n].batch for n in W.CONFIGS},
           "sha256": {n: digests(n) for n in W.CONFIGS}}
    with open(OUT, "w") as f:
        json.dump(man, f, indent=1, sort_keys=True)
        f.write("\n")
    print(OUT)


if __name__ == "__main__":
    main()
