"""CPU oracle for batched TFHE programmable bootstrapping — TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It wraps the plain C oracle in
``tfhe_oracle.c`` (schoolbook negacyclic products mod 2^64, one CMux at a
time) with ctypes and numpy, and spreads independent ciphertexts over host
threads.  It shares no code with the CUDA library.

Every function here follows the construction the paper uses as its TFHE
primitive (Background, "TFHE Scheme": PBS, test polynomial, blind rotation,
extraction of the constant term) plus the standard gadget decomposition and
key switch of the TFHE construction the paper cites.
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tfhe_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_liboracle.so")
_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile the C oracle into oracle/_liboracle.so (gcc, -O2)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < max(
            os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "tfhe_oracle.h"))):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class OrcParams(ctypes.Structure):
    _fields_ = [(name, ctypes.c_uint32) for name in
                ("n", "k", "N", "base_log", "level", "ks_base_log", "ks_level", "msg_bits")]


def _u64p(a: np.ndarray):
    assert a.dtype == np.uint64 and a.flags["C_CONTIGUOUS"], (a.dtype, a.flags)
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_uint64))


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB_PATH)
            P = ctypes.POINTER(ctypes.c_uint64)
            u32 = ctypes.c_uint32
            pp = ctypes.POINTER(OrcParams)
            L.orc_poly_mul.argtypes = [P, P, P, u32]
            L.orc_poly_monomial.argtypes = [P, P, u32, u32]
            L.orc_decompose.argtypes = [ctypes.c_uint64, u32, u32, ctypes.POINTER(ctypes.c_int64)]
            L.orc_modswitch.argtypes = [ctypes.c_uint64, u32]
            L.orc_modswitch.restype = u32
            L.orc_lwe_encrypt.argtypes = [P, P, u32, ctypes.c_uint64, P, ctypes.c_uint64]
            L.orc_lwe_phase.argtypes = [P, P, u32]
            L.orc_lwe_phase.restype = ctypes.c_uint64
            L.orc_decrypt.argtypes = [P, P, u32, u32]
            L.orc_decrypt.restype = ctypes.c_uint64
            L.orc_glwe_encrypt.argtypes = [P, P, u32, u32, P, P, P]
            L.orc_glwe_phase.argtypes = [P, P, P, u32, u32]
            L.orc_ggsw_encrypt.argtypes = [P, P, u32, u32, u32, u32, ctypes.c_uint64, P, P]
            L.orc_bsk_gen.argtypes = [P, pp, P, P, P, P]
            L.orc_ksk_gen.argtypes = [P, pp, P, P, P, P]
            L.orc_test_poly.argtypes = [P, P, u32, u32]
            L.orc_external_product.argtypes = [P, P, P, u32, u32, u32, u32]
            L.orc_cmux_rotate.argtypes = [P, P, u32, u32, u32, u32, u32]
            L.orc_blind_rotate.argtypes = [P, pp, P, P, P]
            L.orc_sample_extract.argtypes = [P, P, u32, u32]
            L.orc_blind_rotate_glwe.argtypes = [P, pp, P, P, P]
            L.orc_automorphism.argtypes = [P, P, u32, u32]
            L.orc_auto_key_gen.argtypes = [P, P, u32, u32, u32, u32, P, P]
            L.orc_trace_step.argtypes = [P, P, u32, u32, u32, u32]
            L.orc_trace.argtypes = [P, P, u32, u32, u32]
            L.orc_plaintext_mul.argtypes = [P, P, P, P, u32]
            L.orc_keyswitch.argtypes = [P, pp, P, P]
            L.orc_blind_rotate_extract.argtypes = [P, pp, P, P, P]
            L.orc_pbs.argtypes = [P, pp, P, P, P, P]
            _lib = L
    return _lib


def params(p) -> OrcParams:
    """OrcParams from a workload.Params (or anything with the same fields)."""
    return OrcParams(p.n, p.k, p.N, p.pbs_base_log, p.pbs_level, p.ks_base_log, p.ks_level, p.msg_bits)


def _c(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.uint64)


def default_threads() -> int:
    return max(1, len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count() or 1)


# ---------------------------------------------------------------- ring / gadget

def poly_mul(a, b) -> np.ndarray:
    a, b = _c(a), _c(b)
    out = np.empty_like(a)
    lib().orc_poly_mul(_u64p(out), _u64p(a), _u64p(b), a.size)
    return out


def poly_monomial(a, u: int) -> np.ndarray:
    a = _c(a)
    out = np.empty_like(a)
    lib().orc_poly_monomial(_u64p(out), _u64p(a), u, a.size)
    return out


def decompose(x: int, base_log: int, level: int) -> list:
    d = (ctypes.c_int64 * level)()
    lib().orc_decompose(ctypes.c_uint64(int(x) & (2**64 - 1)), base_log, level, d)
    return list(d)


def modswitch(x: int, log2_2N: int) -> int:
    return lib().orc_modswitch(ctypes.c_uint64(int(x) & (2**64 - 1)), log2_2N)


# ---------------------------------------------------------------- encryption

def lwe_encrypt(s, msgs, mask, noise) -> np.ndarray:
    """Batch of LWE ciphertexts [count][n+1]; msgs are torus words."""
    s, mask = _c(s), _c(mask)
    msgs, noise = _c(msgs), _c(noise)
    count, n = mask.shape
    out = np.empty((count, n + 1), np.uint64)
    L = lib()
    for b in range(count):
        L.orc_lwe_encrypt(_u64p(out[b]), _u64p(s), n, ctypes.c_uint64(int(msgs[b])), _u64p(mask[b]),
                          ctypes.c_uint64(int(noise[b])))
    return out


def lwe_phase(s, cts) -> np.ndarray:
    s, cts = _c(s), _c(np.atleast_2d(cts))
    n = s.size
    return np.array([lib().orc_lwe_phase(_u64p(cts[b]), _u64p(s), n) for b in range(cts.shape[0])], np.uint64)


def decrypt(s, cts, msg_bits: int) -> np.ndarray:
    s, cts = _c(s), _c(np.atleast_2d(cts))
    n = s.size
    return np.array([lib().orc_decrypt(_u64p(cts[b]), _u64p(s), n, msg_bits) for b in range(cts.shape[0])],
                    np.int64)


def glwe_encrypt(S, msg, mask, noise) -> np.ndarray:
    S, mask, noise = _c(S), _c(mask), _c(noise)
    k, N = S.shape
    out = np.empty((k + 1, N), np.uint64)
    m = _c(msg) if msg is not None else None
    lib().orc_glwe_encrypt(_u64p(out), _u64p(S), k, N, _u64p(m) if m is not None else None,
                           _u64p(mask), _u64p(noise))
    return out


def glwe_phase(S, ct) -> np.ndarray:
    S, ct = _c(S), _c(ct)
    k, N = S.shape
    out = np.empty(N, np.uint64)
    lib().orc_glwe_phase(_u64p(out), _u64p(ct), _u64p(S), k, N)
    return out


def ggsw_encrypt(S, mu: int, base_log: int, level: int, mask, noise) -> np.ndarray:
    S, mask, noise = _c(S), _c(mask), _c(noise)
    k, N = S.shape
    out = np.empty(((k + 1) * level, k + 1, N), np.uint64)
    lib().orc_ggsw_encrypt(_u64p(out), _u64p(S), k, N, base_log, level, ctypes.c_uint64(mu), _u64p(mask),
                           _u64p(noise))
    return out


class Keys:
    """Secret keys plus the raw bootstrapping and key-switching keys."""

    def __init__(self, p, draws, threads: int | None = None):
        self.p = p
        self.lwe_key = _c(draws.lwe_key)
        self.glwe_key = _c(draws.glwe_key)
        self.big_key = self.glwe_key.reshape(-1).copy()    # s'_{jN+t} = S_j[t]
        P = params(p)
        n, k, N, l = p.n, p.k, p.N, p.pbs_level
        self.bsk = np.empty(p.bsk_shape(), np.uint64)
        mask, noise = _c(draws.bsk_mask), _c(draws.bsk_noise)
        rows = (k + 1) * l
        L = lib()
        ggsw_words = rows * (k + 1) * N

        def one(i):
            L.orc_ggsw_encrypt(_u64p(self.bsk[i]), _u64p(self.glwe_key), k, N, p.pbs_base_log, l,
                               ctypes.c_uint64(int(self.lwe_key[i])), _u64p(mask[i]), _u64p(noise[i]))

        with ThreadPoolExecutor(threads or default_threads()) as ex:
            list(ex.map(one, range(n)))
        assert self.bsk[0].size == ggsw_words
        self.ksk = np.empty(p.ksk_shape(), np.uint64)
        L.orc_ksk_gen(_u64p(self.ksk), ctypes.byref(P), _u64p(self.big_key), _u64p(self.lwe_key),
                      _u64p(_c(draws.ksk_mask)), _u64p(_c(draws.ksk_noise)))

    def encrypt(self, cdraws) -> np.ndarray:
        msgs = (np.asarray(cdraws.codes, dtype=np.uint64) << np.uint64(self.p.delta_log2)).astype(np.uint64)
        return lwe_encrypt(self.lwe_key, msgs, cdraws.mask, cdraws.noise)

    def decrypt(self, cts) -> np.ndarray:
        return decrypt(self.lwe_key, cts, self.p.msg_bits)

    def decrypt_big(self, cts) -> np.ndarray:
        return decrypt(self.big_key, cts, self.p.msg_bits)


# ---------------------------------------------------------------- bootstrapping

def test_poly(lut, msg_bits: int, N: int) -> np.ndarray:
    lut = _c(lut)
    v = np.empty(N, np.uint64)
    lib().orc_test_poly(_u64p(v), _u64p(lut), msg_bits, N)
    return v


def external_product(ggsw, glwe, base_log: int, level: int) -> np.ndarray:
    ggsw, glwe = _c(ggsw), _c(glwe)
    kp1, N = glwe.shape
    out = np.empty_like(glwe)
    lib().orc_external_product(_u64p(out), _u64p(ggsw), _u64p(glwe), kp1 - 1, N, base_log, level)
    return out


def cmux_rotate(acc, ggsw, a_tilde: int, base_log: int, level: int) -> np.ndarray:
    acc = _c(acc).copy()
    kp1, N = acc.shape
    lib().orc_cmux_rotate(_u64p(acc), _u64p(_c(ggsw)), a_tilde, kp1 - 1, N, base_log, level)
    return acc


def sample_extract(glwe) -> np.ndarray:
    glwe = _c(glwe)
    kp1, N = glwe.shape
    out = np.empty((kp1 - 1) * N + 1, np.uint64)
    lib().orc_sample_extract(_u64p(out), _u64p(glwe), kp1 - 1, N)
    return out


def _batch(fn_name, out_words, p, bsk_or_none, ksk_or_none, lwe, lut, threads):
    L = lib()
    P = params(p)
    lwe = _c(np.atleast_2d(lwe))
    lut = _c(lut)
    out = np.empty((lwe.shape[0], out_words), np.uint64)
    fn = getattr(L, fn_name)
    bsk = _c(bsk_or_none) if bsk_or_none is not None else None
    ksk = _c(ksk_or_none) if ksk_or_none is not None else None

    def one(b):
        if fn_name == "orc_pbs":
            fn(_u64p(out[b]), ctypes.byref(P), _u64p(bsk), _u64p(ksk), _u64p(lwe[b]), _u64p(lut))
        else:
            fn(_u64p(out[b]), ctypes.byref(P), _u64p(bsk), _u64p(lwe[b]), _u64p(lut))

    t = threads or default_threads()
    if t == 1 or lwe.shape[0] == 1:
        for b in range(lwe.shape[0]):
            one(b)
    else:
        with ThreadPoolExecutor(t) as ex:
            list(ex.map(one, range(lwe.shape[0])))
    return out


def blind_rotate(p, bsk, lwe, lut) -> np.ndarray:
    """GLWE accumulator [(k+1)][N] after blind rotation of one LWE."""
    L = lib()
    P = params(p)
    acc = np.empty((p.k + 1, p.N), np.uint64)
    L.orc_blind_rotate(_u64p(acc), ctypes.byref(P), _u64p(_c(bsk)), _u64p(_c(lwe)), _u64p(_c(lut)))
    return acc


def blind_rotate_glwe_batch(p, bsk, lwe, glwe_in, threads=None) -> np.ndarray:
    """[batch][(k+1)][N]: blind rotation of each ciphertext's own GLWE test
    polynomial glwe_in[b] by the phase of lwe[b]."""
    L = lib()
    P = params(p)
    lwe = _c(np.atleast_2d(lwe))
    glwe_in = _c(glwe_in).reshape(lwe.shape[0], p.k + 1, p.N)
    bsk = _c(bsk)
    out = np.empty_like(glwe_in)

    def one(b):
        L.orc_blind_rotate_glwe(_u64p(out[b]), ctypes.byref(P), _u64p(bsk), _u64p(lwe[b]), _u64p(glwe_in[b]))

    with ThreadPoolExecutor(threads or default_threads()) as ex:
        list(ex.map(one, range(lwe.shape[0])))
    return out


# ---------------------------------------------------------------- RLWE trace (k = 1)

def automorphism(a, k: int) -> np.ndarray:
    a = _c(a)
    out = np.empty_like(a)
    lib().orc_automorphism(_u64p(out), _u64p(a), k, a.size)
    return out


def trace_exponents(N: int) -> list:
    """Automorphism exponents of the trace steps, in order: N+1, N/2+1, ..., 3."""
    logN = N.bit_length() - 1
    return [(1 << (logN - s)) + 1 for s in range(logN)]


def trace_keys(S, base_log: int, level: int, mask, noise) -> np.ndarray:
    """[log2 N][level][2][N] automorphism keys; mask/noise [log2 N][level][N]."""
    S = _c(S).reshape(-1)
    N = S.size
    ks = trace_exponents(N)
    out = np.empty((len(ks), level, 2, N), np.uint64)
    mask, noise = _c(mask), _c(noise)
    for s, k in enumerate(ks):
        lib().orc_auto_key_gen(_u64p(out[s]), _u64p(S), N, k, base_log, level, _u64p(mask[s]), _u64p(noise[s]))
    return out


def trace_batch(keys, glwe, base_log: int, level: int, threads=None) -> np.ndarray:
    """[batch][2][N] traces of GLWE ciphertexts (k = 1)."""
    keys = _c(keys)
    out = _c(glwe).copy()
    N = out.shape[-1]

    def one(b):
        lib().orc_trace(_u64p(out[b]), _u64p(keys), N, base_log, level)

    with ThreadPoolExecutor(threads or default_threads()) as ex:
        list(ex.map(one, range(out.shape[0])))
    return out


def plaintext_mul_batch(glwe, plain_mul, plain_add=None) -> np.ndarray:
    """[batch][2][N]: (P * A, P * B + Q) for each GLWE; P given as signed ints."""
    glwe = _c(glwe)
    P = np.asarray(plain_mul, dtype=np.int64).view(np.uint64).copy()
    Qp = _c(plain_add) if plain_add is not None else None
    out = np.empty_like(glwe)
    N = glwe.shape[-1]
    for b in range(glwe.shape[0]):
        lib().orc_plaintext_mul(_u64p(out[b]), _u64p(glwe[b]), _u64p(P), _u64p(Qp) if Qp is not None else None, N)
    return out


def pbs_batch_multi_lut(p, bsk, ksk, lwe, luts, lut_index, threads=None) -> np.ndarray:
    """PBS of ciphertext b with LUT luts[lut_index[b]]."""
    lwe = _c(np.atleast_2d(lwe))
    luts = _c(luts)
    out = np.empty((lwe.shape[0], p.n + 1), np.uint64)
    for li in np.unique(lut_index):
        sel = np.nonzero(np.asarray(lut_index) == li)[0]
        out[sel] = pbs_batch(p, bsk, ksk, lwe[sel], luts[li], threads)
    return out


def blind_rotate_extract_batch(p, bsk, lwe, lut, threads=None) -> np.ndarray:
    return _batch("orc_blind_rotate_extract", p.k * p.N + 1, p, bsk, None, lwe, lut, threads)


def pbs_batch(p, bsk, ksk, lwe, lut, threads=None) -> np.ndarray:
    """[batch][n+1] outputs of PBS (modswitch, blind rotation, extraction,
    key switch) for each input LWE ciphertext."""
    return _batch("orc_pbs", p.n + 1, p, bsk, ksk, lwe, lut, threads)


def keyswitch_batch(p, ksk, lwe_big, threads=None) -> np.ndarray:
    L = lib()
    P = params(p)
    lwe_big = _c(np.atleast_2d(lwe_big))
    ksk = _c(ksk)
    out = np.empty((lwe_big.shape[0], p.n + 1), np.uint64)

    def one(b):
        L.orc_keyswitch(_u64p(out[b]), ctypes.byref(P), _u64p(ksk), _u64p(lwe_big[b]))

    with ThreadPoolExecutor(threads or default_threads()) as ex:
        list(ex.map(one, range(lwe_big.shape[0])))
    return out


# ---------------------------------------------------------------- encrypted segmented lookup (k = 1)

def segment_box(s: int, n_seg: int, N: int) -> np.ndarray:
    """[N] int64: +1 on the coefficients s N/n_seg + d, -h <= d < h (h half a
    box), the ones below 0 wrapped to N + d with a minus sign (X^N = -1)."""
    box = N // n_seg
    h = box // 2
    v = np.zeros(N, np.int64)
    for d in range(-h, box - h):
        j = s * box + d
        if j < 0:
            v[j + N] = -1
        else:
            v[j] = 1
    return v


def segmented_lookup_batch(p, bsk, ksk, tkeys, t_base_log: int, t_level: int, glwe_x, lwe_seg,
                           p_hat, q_hat, a_hat, b_hat, threads=None) -> np.ndarray:
    """[batch][2][N]: the encrypted lookup of the Cryptographic Lookup
    Protocol, Steps 2 and 3, for each [[x]] (glwe_x) and segment index [[S]]
    (lwe_seg), with the caller's integer tables.
      Step 2: [[t]] = p [[x]] + q; PBS([[t]], [[S]]) (blind rotation,
              extraction of the constant term, key switch) = [[I]].
      Step 3, phase 1: [[r_s]] = a_s [[x]] + b_s; r_s = Trace(BlindRot(r_s, [[I]])).
      Phase 2: [[R]] = sum_s r_s X^s, the s-th coefficient being the segment
              box of s (so r_s times the box polynomial);
              out = Trace(BlindRot([[R]], [[S]]))."""
    glwe_x = _c(glwe_x)
    lwe_seg = _c(np.atleast_2d(lwe_seg))
    batch, _, N = glwe_x.shape
    n_seg = a_hat.shape[0]
    # Step 2
    t = plaintext_mul_batch(glwe_x, p_hat, q_hat)
    t_rot = blind_rotate_glwe_batch(p, bsk, lwe_seg, t, threads)
    lwe_I = keyswitch_batch(p, ksk, np.stack([sample_extract(g) for g in t_rot]), threads)
    # Step 3, phase 1 (all segments of all ciphertexts at once)
    r = np.concatenate([plaintext_mul_batch(glwe_x, a_hat[s], b_hat[s]) for s in range(n_seg)])
    r = blind_rotate_glwe_batch(p, bsk, np.tile(lwe_I, (n_seg, 1)), r, threads)
    r = trace_batch(tkeys, r, t_base_log, t_level, threads).reshape(n_seg, batch, 2, N)
    # phase 2
    R = np.zeros((batch, 2, N), np.uint64)
    for s in range(n_seg):
        R += plaintext_mul_batch(r[s], segment_box(s, n_seg, N))
    R_rot = blind_rotate_glwe_batch(p, bsk, lwe_seg, R, threads)
    return trace_batch(tkeys, R_rot, t_base_log, t_level, threads)
