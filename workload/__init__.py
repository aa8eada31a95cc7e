"""Seeded synthetic workloads for batched TFHE programmable bootstrapping.

This module only draws random numbers and defines the workload shapes; it
holds none of the scheme's arithmetic (no encryption, no key generation, no
polynomial products).  Both the CPU oracle (``oracle/``) and the CUDA path's
tests and benchmark take their inputs from here.

Parameter sets follow the paper's use of PBS for the nonlinear layers of LLM
decoding (Background, "TFHE Scheme": PBS evaluates a LUT f on an LWE
ciphertext; Evaluation, "Experimental Setup": LUT precision, ranges).  The
torus is Z_{2^64}; every ciphertext word is a uint64.

Randomness: numpy's PCG64 bit generator (O'Neill 2014) seeded through a
SeedSequence([master_seed, purpose]); only its raw 64-bit outputs are used,
whose stream numpy keeps fixed across versions and platforms.  Uniform words
are raw outputs.  Normal variates are the Irwin-Hall sum of twelve uniforms
minus six (mean 0, variance 1, tails cut at 6 sigma), formed in integer
arithmetic from the top 53 bits of twelve raw outputs, so every draw is the
same on every host; Gaussian noise is that variate times 2^sigma_log2,
rounded half up to an integer, stored as two's complement.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

# --------------------------------------------------------------------------
# parameter sets
# --------------------------------------------------------------------------


@dataclass(frozen=True)
class Params:
    """One PBS parameter set (torus q = 2^64, one padding bit)."""

    name: str
    n: int                 # LWE dimension of input/output ciphertexts
    k: int                 # GLWE dimension
    N: int                 # GLWE polynomial size (power of two)
    pbs_base_log: int      # beta: PBS gadget base 2^beta
    pbs_level: int         # ell: PBS gadget levels
    ks_base_log: int       # beta_ks
    ks_level: int          # ell_ks
    msg_bits: int          # p: LUT has 2^p entries
    lwe_sigma_log2: int    # LWE noise std = 2^lwe_sigma_log2 (integer torus units)
    glwe_sigma_log2: int   # GLWE/GGSW noise std
    lut: tuple             # ("square_mod", ) or (kind, lo, hi)
    msg: tuple             # ("uniform",) or ("normal", std, lo, hi)
    batch: int             # headline batch size
    seed: int
    batches: tuple = field(default_factory=tuple)

    @property
    def delta_log2(self) -> int:
        return 63 - self.msg_bits

    @property
    def kN(self) -> int:
        return self.k * self.N

    def bsk_shape(self):
        return (self.n, (self.k + 1) * self.pbs_level, self.k + 1, self.N)

    def ksk_shape(self):
        return (self.kN, self.ks_level, self.n + 1)


CONFIGS = {
    # Tiny PBS: n=64, k=1, N=256, PBS 2^10 x 2, KS 2^4 x 4, sigma = 2^-40 of the
    # torus (2^24 integer), 3-bit messages, LUT m -> m^2 mod 8, batch 16.
    "tiny": Params("tiny", n=64, k=1, N=256, pbs_base_log=10, pbs_level=2,
                   ks_base_log=4, ks_level=4, msg_bits=3, lwe_sigma_log2=24,
                   glwe_sigma_log2=24, lut=("square_mod",), msg=("uniform",),
                   batch=16, seed=1),
    # Standard-size PBS: n=742, N=2048, PBS 2^23 x 1, KS 2^3 x 5,
    # sigma_lwe = 2^-17, sigma_glwe = 2^-51, 4-bit GELU on [-4, 4], batch 4096.
    "standard": Params("standard", n=742, k=1, N=2048, pbs_base_log=23, pbs_level=1,
                       ks_base_log=3, ks_level=5, msg_bits=4, lwe_sigma_log2=47,
                       glwe_sigma_log2=13, lut=("gelu", -4.0, 4.0), msg=("uniform",),
                       batch=4096, seed=2),
    # GPT-2-small MLP nonlinearity: 3072 activations, N(0,1) clipped [-4,4],
    # 6-bit GELU; n=840, N=4096, PBS 2^15 x 2, KS 2^4 x 5.
    "gpt2_mlp": Params("gpt2_mlp", n=840, k=1, N=4096, pbs_base_log=15, pbs_level=2,
                       ks_base_log=4, ks_level=5, msg_bits=6, lwe_sigma_log2=42,
                       glwe_sigma_log2=13, lut=("gelu", -4.0, 4.0),
                       msg=("normal", 1.0, -4.0, 4.0), batch=3072, seed=3),
    # LLaMA-3-8B SiLU: 14336 activations, N(0,1.5) clipped [-6,6], 7-bit SiLU;
    # n=900, N=8192, PBS 2^14 x 3, KS 2^4 x 6.
    "llama_silu": Params("llama_silu", n=900, k=1, N=8192, pbs_base_log=14, pbs_level=3,
                         ks_base_log=4, ks_level=6, msg_bits=7, lwe_sigma_log2=42,
                         glwe_sigma_log2=13, lut=("silu", -6.0, 6.0),
                         msg=("normal", 1.5, -6.0, 6.0), batch=14336, seed=4),
    # Softmax-logit sweep at the standard parameters: 5-bit exp on [-8, 0],
    # N(0,2) clipped to [-8, 0]; batch 1 .. 65536.
    "exp_sweep": Params("exp_sweep", n=742, k=1, N=2048, pbs_base_log=23, pbs_level=1,
                        ks_base_log=3, ks_level=5, msg_bits=5, lwe_sigma_log2=47,
                        glwe_sigma_log2=13, lut=("exp", -8.0, 0.0),
                        msg=("normal", 2.0, -8.0, 0.0), batch=1024, seed=5,
                        batches=(1, 64, 1024, 16384, 65536)),
    # The paper's TFHE dimensions (n = 1024, N_br = 2048; Experimental Setup)
    # on the 2^64 torus: PBS 2^23 x 1, KS 2^3 x 5, 4-bit GELU, batch 4096.
    "paper_dims": Params("paper_dims", n=1024, k=1, N=2048, pbs_base_log=23, pbs_level=1,
                         ks_base_log=3, ks_level=5, msg_bits=4, lwe_sigma_log2=47,
                         glwe_sigma_log2=13, lut=("gelu", -4.0, 4.0), msg=("uniform",),
                         batch=4096, seed=7),
    # Encrypted segmented lookup on a small ring (two traces multiply the
    # result by N^2, so the noise of a blind rotation must stay well below
    # 2^63 / N^2): n=64, N=512, PBS 2^8 x 6, KS 2^4 x 8, 1/x on [0.1, 2.0]
    # with the paper's two segments and four intervals per segment.
    "lookup_small": Params("lookup_small", n=64, k=1, N=512, pbs_base_log=8, pbs_level=6,
                           ks_base_log=4, ks_level=8, msg_bits=2, lwe_sigma_log2=30,
                           glwe_sigma_log2=13, lut=("reciprocal", 0.1, 2.0),
                           msg=("uniform",), batch=8, seed=6),
}

# purposes of independent random streams
_PURPOSE = {
    "lwe_key": 1, "glwe_key": 2, "bsk_mask": 3, "bsk_noise": 4, "ksk_mask": 5,
    "ksk_noise": 6, "ct_mask": 7, "ct_noise": 8, "messages": 9, "uniform_keys": 10,
    "uniform_cts": 11, "sample": 12, "trace_mask": 13, "trace_noise": 14, "glwe_mask": 15,
    "glwe_noise": 16, "inputs": 17,
}


def rng(seed: int, purpose: str, sub: int = 0) -> np.random.Generator:
    """Independent stream for (master seed, purpose, sub-seed)."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, _PURPOSE[purpose], sub])))


def uniform_u64(shape, g: np.random.Generator) -> np.ndarray:
    count = int(np.prod(shape))
    return g.bit_generator.random_raw(count).astype(np.uint64).reshape(shape)


def binary_u64(shape, g: np.random.Generator) -> np.ndarray:
    return (uniform_u64(shape, g) >> np.uint64(63)).astype(np.uint64)


_IH_TERMS = 12      # uniforms per normal variate
_IH_BITS = 53       # bits kept of each raw output


def normal_fixed(count: int, g: np.random.Generator) -> np.ndarray:
    """Approximately standard normal variates as exact integers z * 2^53:
    the sum of twelve uniform 53-bit integers minus 6 * 2^53 (Irwin-Hall:
    mean 0, variance 1, |z| < 6), int64."""
    u = (g.bit_generator.random_raw(_IH_TERMS * count).astype(np.uint64) >> np.uint64(64 - _IH_BITS)).astype(np.int64)
    return u.reshape(count, _IH_TERMS).sum(axis=1) - np.int64(6 << _IH_BITS)


def standard_normal(count: int, g: np.random.Generator) -> np.ndarray:
    """The same variates as float64 (z * 2^53 rounded to 53 bits, then
    scaled by 2^-53: IEEE arithmetic, identical on every host)."""
    return normal_fixed(count, g).astype(np.float64) * (2.0 ** -_IH_BITS)


def gaussian_u64(shape, sigma_log2: int, g: np.random.Generator) -> np.ndarray:
    """round(2^sigma_log2 * z) (ties up), z from normal_fixed, as
    two's-complement uint64; exact integer arithmetic (sigma_log2 < 53)."""
    assert 0 <= sigma_log2 < _IH_BITS
    zf = normal_fixed(int(np.prod(shape)), g)
    sh = _IH_BITS - sigma_log2
    v = (zf + np.int64(1 << (sh - 1))) >> np.int64(sh)      # arithmetic shift: floor
    return v.astype(np.int64).view(np.uint64).reshape(shape)


# --------------------------------------------------------------------------
# LUTs and messages
# --------------------------------------------------------------------------


def _gelu(x: float) -> float:
    return 0.5 * x * (1.0 + math.erf(x / math.sqrt(2.0)))


def _silu(x: float) -> float:
    return x / (1.0 + math.exp(-x))


def bin_midpoints(lo: float, hi: float, entries: int) -> list:
    """Staircase LUT: each of `entries` equal intervals of [lo, hi] is
    represented by its midpoint (Segmented LUT Evaluation, single-LUT
    construction)."""
    w = (hi - lo) / entries
    return [lo + (m + 0.5) * w for m in range(entries)]


def bin_index(x: float, lo: float, hi: float, entries: int) -> int:
    """I = floor((x - lo) / (hi - lo) * entries), clamped to the table."""
    i = math.floor((x - lo) / (hi - lo) * entries)
    return min(max(i, 0), entries - 1)


def lut_codes(params: Params) -> np.ndarray:
    """Output codes (integers in [0, 2^p)) of the LUT for each input code."""
    p = params.msg_bits
    size = 1 << p
    if params.lut[0] == "square_mod":
        return np.array([(m * m) % size for m in range(size)], dtype=np.int64)
    kind, lo, hi = params.lut
    f = {"gelu": _gelu, "silu": _silu, "exp": math.exp, "reciprocal": lambda x: 1.0 / x}[kind]
    ys = [f(x) for x in bin_midpoints(lo, hi, size)]
    y_lo, y_hi = min(ys), max(ys)
    codes = [min(max(math.floor((y - y_lo) / (y_hi - y_lo) * (size - 1) + 0.5), 0), size - 1) for y in ys]
    return np.array(codes, dtype=np.int64)


def lut_torus(params: Params, codes=None) -> np.ndarray:
    """LUT entries as torus words Delta * code, Delta = 2^(63 - p)."""
    if codes is None:
        codes = lut_codes(params)
    return (np.asarray(codes, dtype=np.uint64) << np.uint64(params.delta_log2)).astype(np.uint64)


def message_codes(params: Params, count: int, g: np.random.Generator) -> np.ndarray:
    """Input codes in [0, 2^p) with the workload's value distribution."""
    size = 1 << params.msg_bits
    if params.msg[0] == "uniform":
        return (uniform_u64((count,), g) % np.uint64(size)).astype(np.int64)
    _, std, lo, hi = params.msg
    x = np.clip(standard_normal(count, g) * std, lo, hi)
    m = np.floor((x - lo) / (hi - lo) * size).astype(np.int64)
    return np.clip(m, 0, size - 1)


# --------------------------------------------------------------------------
# draws consumed by key generation and encryption
# --------------------------------------------------------------------------


@dataclass
class KeyDraws:
    """Every random value key generation needs; zero masks/noise give the
    trivial (noiseless, unmasked) keys used by closed-form tests."""

    lwe_key: np.ndarray      # [n] in {0,1}
    glwe_key: np.ndarray     # [k][N] in {0,1}
    bsk_mask: np.ndarray     # [n][(k+1)l][k][N]
    bsk_noise: np.ndarray    # [n][(k+1)l][N]
    ksk_mask: np.ndarray     # [kN][l_ks][n]
    ksk_noise: np.ndarray    # [kN][l_ks]


def key_draws(params: Params, seed=None, trivial: bool = False) -> KeyDraws:
    s = params.seed if seed is None else seed
    n, k, N, l, lk = params.n, params.k, params.N, params.pbs_level, params.ks_level
    lwe_key = binary_u64((n,), rng(s, "lwe_key"))
    glwe_key = binary_u64((k, N), rng(s, "glwe_key"))
    if trivial:
        return KeyDraws(lwe_key, glwe_key,
                        np.zeros((n, (k + 1) * l, k, N), np.uint64), np.zeros((n, (k + 1) * l, N), np.uint64),
                        np.zeros((k * N, lk, n), np.uint64), np.zeros((k * N, lk), np.uint64))
    return KeyDraws(
        lwe_key, glwe_key,
        uniform_u64((n, (k + 1) * l, k, N), rng(s, "bsk_mask")),
        gaussian_u64((n, (k + 1) * l, N), params.glwe_sigma_log2, rng(s, "bsk_noise")),
        uniform_u64((k * N, lk, n), rng(s, "ksk_mask")),
        gaussian_u64((k * N, lk), params.lwe_sigma_log2, rng(s, "ksk_noise")),
    )


@dataclass
class CipherDraws:
    codes: np.ndarray   # [batch] message codes
    mask: np.ndarray    # [batch][n]
    noise: np.ndarray   # [batch]


def cipher_draws(params: Params, count: int, seed=None, sub: int = 0, codes=None) -> CipherDraws:
    s = params.seed if seed is None else seed
    if codes is None:
        codes = message_codes(params, count, rng(s, "messages", sub))
    return CipherDraws(
        np.asarray(codes, dtype=np.int64),
        uniform_u64((count, params.n), rng(s, "ct_mask", sub)),
        gaussian_u64((count,), params.lwe_sigma_log2, rng(s, "ct_noise", sub)),
    )


def uniform_keys(params: Params, seed=None):
    """Raw BSK and KSK of uniform words.  A real key (GLWE/LWE encryptions
    under a secret) is indistinguishable from uniform words, and the cost of
    PBS does not depend on the key values, so timing runs may use these."""
    s = params.seed if seed is None else seed
    g = rng(s, "uniform_keys")
    return uniform_u64(params.bsk_shape(), g), uniform_u64(params.ksk_shape(), g)


def uniform_ciphertexts(params: Params, count: int, seed=None, sub: int = 0) -> np.ndarray:
    s = params.seed if seed is None else seed
    return uniform_u64((count, params.n + 1), rng(s, "uniform_cts", sub))
