"""Helpers shared by the GPU tests: device buffers and contexts."""

import numpy as np

import paper_2609_16915_gb300 as R


def torch():
    import torch as _t
    return _t


def to_dev(a: np.ndarray):
    t = torch()
    return t.from_numpy(np.ascontiguousarray(a, dtype=np.uint64).view(np.int64)).cuda()


def to_host(t) -> np.ndarray:
    return t.cpu().numpy().view(np.uint64)


def empty_dev(*shape):
    t = torch()
    return t.empty(shape, dtype=t.int64, device="cuda")


def make_ctx(p, bsk, ksk, max_batch=0):
    ctx = R.Context(p, device=0, max_batch=max_batch)
    ctx.upload_bsk(to_dev(bsk))
    ctx.upload_ksk(to_dev(ksk))
    ctx.sync_status()
    return ctx


def gpu_pbs(ctx, p, lwe, lut):
    out = empty_dev(lwe.shape[0], p.n + 1)
    ctx.pbs_batch(to_dev(lwe), to_dev(lut), out)
    ctx.sync_status()
    return to_host(out)


def gpu_br_extract(ctx, p, lwe, lut):
    out = empty_dev(lwe.shape[0], p.kN + 1)
    ctx.blind_rotate_extract_batch(to_dev(lwe), to_dev(lut), out)
    ctx.sync_status()
    return to_host(out)


def gpu_keyswitch(ctx, p, big):
    out = empty_dev(big.shape[0], p.n + 1)
    ctx.keyswitch_batch(to_dev(big), out)
    ctx.sync_status()
    return to_host(out)


def sparse_lwe(p, count, nonzero, seed):
    """LWE words with all but `nonzero` mask words zero: blind rotation then
    runs only that many CMux steps (a~_i = 0 steps add nothing), so the
    oracle can check full-size parameters quickly."""
    g = np.random.default_rng(seed)
    lwe = np.zeros((count, p.n + 1), np.uint64)
    for b in range(count):
        idx = g.choice(p.n, size=nonzero, replace=False)
        lwe[b, idx] = g.integers(0, 2**64, size=nonzero, dtype=np.uint64, endpoint=False)
        lwe[b, p.n] = g.integers(0, 2**64, dtype=np.uint64, endpoint=False)
    return lwe
