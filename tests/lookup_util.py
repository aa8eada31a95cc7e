"""Shared setup of the encrypted segmented-lookup tests: keys, trace keys,
encoded tables and encrypted inputs, all from the oracle and seeded draws."""

import numpy as np

import oracle as O
import workload as W
from paper_2609_16915_gb300 import segmented as SG

TRACE_BASE_LOG, TRACE_LEVEL = 8, 8   # exact 64-bit gadget, small digits (low trace noise)
# scales of x and of the values a x + b before the traces: slopes are carried as
# round(a 2^(DR - DX)), x with the GLWE noise 2^13 at 2^-19 of a unit, and
# N^2 2^DR |f| stays below 2^63 for N = 512 and |f| <= 10
DX, DR = 32, 40


def paper_table():
    """1/x on [0.1, 2.0], boundaries 0.1 | 0.5 | 2.0, four intervals per segment."""
    return SG.build(SG.FUNCTIONS["reciprocal"], [0.1, 0.5, 2.0], 4)


def trace_keys(p, S, base_log=TRACE_BASE_LOG, level=TRACE_LEVEL, noiseless=False, seed=None):
    s = p.seed if seed is None else seed
    steps = p.N.bit_length() - 1
    mask = W.uniform_u64((steps, level, p.N), W.rng(s, "trace_mask"))
    noise = W.gaussian_u64((steps, level, p.N), p.glwe_sigma_log2, W.rng(s, "trace_noise"))
    if noiseless:
        mask[:] = 0
        noise[:] = 0
    return O.trace_keys(S.reshape(-1), base_log, level, mask, noise)


def encrypt_inputs(p, keys, xs, segs, n_seg, dx=DX, sub=0):
    """[[x]] as GLWE (x in the constant coefficient) and [[S]] as LWE."""
    b = len(xs)
    S = keys.glwe_key.reshape(1, -1)
    gmask = W.uniform_u64((b, 1, p.N), W.rng(p.seed, "glwe_mask", sub))
    gnoise = W.gaussian_u64((b, p.N), p.glwe_sigma_log2, W.rng(p.seed, "glwe_noise", sub))
    glwe = np.empty((b, 2, p.N), np.uint64)
    for i, x in enumerate(xs):
        msg = np.zeros(p.N, np.uint64)
        msg[0] = np.uint64(SG.encode_x(x, dx))
        glwe[i] = O.glwe_encrypt(S, msg, gmask[i], gnoise[i])
    words = np.array([SG.segment_word(int(s), n_seg) for s in segs], np.uint64)
    lmask = W.uniform_u64((b, p.n), W.rng(p.seed, "ct_mask", 100 + sub))
    lnoise = W.gaussian_u64((b,), p.lwe_sigma_log2, W.rng(p.seed, "ct_noise", 100 + sub))
    lwe = O.lwe_encrypt(keys.lwe_key, words, lmask, lnoise)
    return glwe, lwe


def sample_points(lut, count, seed):
    """x in the table's domain, kept 2 % of an interval away from every interval edge."""
    g = np.random.default_rng(seed)
    xs = []
    while len(xs) < count:
        x = float(g.uniform(lut.tau[0], lut.tau[-1]))
        s = SG.segment_index(lut, x)
        pos = (x - lut.tau[s]) / (lut.tau[s + 1] - lut.tau[s]) * lut.n_br
        if min(pos - np.floor(pos), np.ceil(pos) - pos) > 0.02:
            xs.append(x)
    return xs
