"""Python binding of librosetta, the sm_103a batched TFHE PBS library.

Argument marshalling only: every step of bootstrapping runs in the CUDA
kernels behind the C ABI declared in include/rosetta.h.  The functions keep
the C names; buffers may be torch tensors (CUDA or CPU) or numpy arrays, and
streams torch streams.  Importing this package does not load the library;
the first call does, and raises if librosetta.so has not been built — there
is no CPU fallback.
"""

from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "librosetta.so")
# the same library compiled with -DROSETTA_DEBUG (device-side bounds checks)
DEBUG_LIB_PATH = os.path.join(_HERE, "librosetta_debug.so")

ROSETTA_OK = 0
STATUS = {0: "ok", -1: "invalid argument", -2: "unsupported parameters", -3: "keys not uploaded",
          -4: "CUDA error", -5: "out of device memory", -6: "device wait timed out",
          -7: "device-side bounds check failed (debug build)"}

EXPORTS = ("rosetta_params_init", "rosetta_upload_bsk", "rosetta_upload_ksk", "rosetta_pbs_batch",
           "rosetta_blind_rotate_extract_batch", "rosetta_keyswitch_batch", "rosetta_pbs_batch_multi_lut",
           "rosetta_blind_rotate_glwe_batch", "rosetta_upload_trace_keys", "rosetta_trace_batch",
           "rosetta_plaintext_mul_batch", "rosetta_upload_lookup_table", "rosetta_segmented_lookup_batch",
           "rosetta_selftest_wait_timeout", "rosetta_selftest_bounds",
           "rosetta_pbs_batch_noalloc", "rosetta_ntt_primes",
           "rosetta_sync_status", "rosetta_destroy", "rosetta_status_string")


class RosettaError(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn} failed: {STATUS.get(status, 'unknown')} ({status})")
        self.status = status


class rosetta_params(ctypes.Structure):
    _fields_ = [(f, ctypes.c_uint32) for f in ("lwe_dim", "glwe_dim", "poly_size", "pbs_base_log", "pbs_level",
                                               "ks_base_log", "ks_level", "msg_bits", "max_batch")]


_lib = None


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load librosetta.so (built by paper_2609_16915_gb300.build)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`"
                           " (the CUDA library is required; there is no CPU fallback)")
    L = ctypes.CDLL(path)
    vp, u32, u64p = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_void_p
    L.rosetta_params_init.argtypes = [ctypes.POINTER(vp), ctypes.POINTER(rosetta_params), ctypes.c_int]
    L.rosetta_upload_bsk.argtypes = [vp, u64p, ctypes.c_size_t, ctypes.c_int, vp]
    L.rosetta_upload_ksk.argtypes = [vp, u64p, ctypes.c_size_t, ctypes.c_int, vp]
    L.rosetta_pbs_batch.argtypes = [vp, u64p, u32, u64p, u64p, vp]
    L.rosetta_blind_rotate_extract_batch.argtypes = [vp, u64p, u32, u64p, u64p, vp]
    L.rosetta_keyswitch_batch.argtypes = [vp, u64p, u32, u64p, vp]
    L.rosetta_pbs_batch_noalloc.argtypes = [vp, u64p, u32, u64p, u64p, vp]
    L.rosetta_pbs_batch_multi_lut.argtypes = [vp, u64p, u32, u64p, u32, vp, u64p, vp]
    L.rosetta_blind_rotate_glwe_batch.argtypes = [vp, u64p, u32, u64p, u64p, vp]
    L.rosetta_upload_trace_keys.argtypes = [vp, u64p, ctypes.c_size_t, u32, u32, ctypes.c_int, vp]
    L.rosetta_trace_batch.argtypes = [vp, u64p, u32, u64p, vp]
    L.rosetta_plaintext_mul_batch.argtypes = [vp, u64p, u32, u64p, u64p, u64p, vp]
    L.rosetta_upload_lookup_table.argtypes = [vp, u32, u64p, u64p, u64p, u64p, vp]
    L.rosetta_segmented_lookup_batch.argtypes = [vp, u64p, u64p, u32, u64p, vp]
    L.rosetta_selftest_wait_timeout.argtypes = [vp, u32, vp]
    L.rosetta_selftest_bounds.argtypes = [vp, vp]
    L.rosetta_ntt_primes.argtypes = [vp]
    L.rosetta_sync_status.argtypes = [vp, vp]
    L.rosetta_destroy.argtypes = [vp]
    L.rosetta_destroy.restype = None
    L.rosetta_status_string.argtypes = [ctypes.c_int]
    L.rosetta_status_string.restype = ctypes.c_char_p
    for name in EXPORTS:
        if name not in ("rosetta_destroy", "rosetta_status_string"):
            getattr(L, name).restype = ctypes.c_int
    _lib = L
    return L


def _ptr(buf) -> int:
    """Address of a torch tensor or numpy array (must be contiguous)."""
    if hasattr(buf, "data_ptr"):
        if not buf.is_contiguous():
            raise ValueError("buffer must be contiguous")
        return buf.data_ptr()
    if not buf.flags["C_CONTIGUOUS"]:
        raise ValueError("buffer must be contiguous")
    return buf.ctypes.data


def _is_device(buf) -> bool:
    return bool(getattr(buf, "is_cuda", False))


def _stream(stream) -> int | None:
    if stream is None:
        try:
            import torch
            if torch.cuda.is_available():
                return torch.cuda.current_stream().cuda_stream
        except ImportError:
            pass
        return None
    return getattr(stream, "cuda_stream", stream)


def _check(fn: str, st: int):
    if st != ROSETTA_OK:
        raise RosettaError(fn, st)


def rosetta_status_string(status: int) -> str:
    return load().rosetta_status_string(status).decode()


class Context:
    """One parameter set on one device: keys, tables and scratch live here."""

    def __init__(self, params, device: int = 0, max_batch: int = 0):
        L = load()
        prm = rosetta_params(params.n, params.k, params.N, params.pbs_base_log, params.pbs_level,
                             params.ks_base_log, params.ks_level, params.msg_bits, max_batch)
        h = ctypes.c_void_p()
        _check("rosetta_params_init", L.rosetta_params_init(ctypes.byref(h), ctypes.byref(prm), device))
        self._h = h
        self.params = params
        self.device = device

    def close(self):
        if getattr(self, "_h", None):
            load().rosetta_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ---- the C entry points ----
    def rosetta_upload_bsk(self, bsk, stream=None):
        n = bsk.numel() if hasattr(bsk, "numel") else bsk.size
        _check("rosetta_upload_bsk", load().rosetta_upload_bsk(self._h, _ptr(bsk), n, int(_is_device(bsk)),
                                                               _stream(stream)))

    def rosetta_upload_ksk(self, ksk, stream=None):
        n = ksk.numel() if hasattr(ksk, "numel") else ksk.size
        _check("rosetta_upload_ksk", load().rosetta_upload_ksk(self._h, _ptr(ksk), n, int(_is_device(ksk)),
                                                               _stream(stream)))

    def rosetta_pbs_batch(self, lwe_in, lut, lwe_out, stream=None):
        batch = lwe_in.shape[0]
        _check("rosetta_pbs_batch", load().rosetta_pbs_batch(self._h, _ptr(lwe_in), batch, _ptr(lut),
                                                             _ptr(lwe_out), _stream(stream)))
        return lwe_out

    def rosetta_blind_rotate_extract_batch(self, lwe_in, lut, lwe_big_out, stream=None):
        batch = lwe_in.shape[0]
        _check("rosetta_blind_rotate_extract_batch",
               load().rosetta_blind_rotate_extract_batch(self._h, _ptr(lwe_in), batch, _ptr(lut), _ptr(lwe_big_out),
                                                         _stream(stream)))
        return lwe_big_out

    def rosetta_keyswitch_batch(self, lwe_big_in, lwe_out, stream=None):
        batch = lwe_big_in.shape[0]
        _check("rosetta_keyswitch_batch", load().rosetta_keyswitch_batch(self._h, _ptr(lwe_big_in), batch,
                                                                         _ptr(lwe_out), _stream(stream)))
        return lwe_out

    def rosetta_pbs_batch_multi_lut(self, lwe_in, luts, lut_index, lwe_out, stream=None):
        """PBS with a LUT per ciphertext: luts [num_luts][2^p], lut_index [batch] (uint32 / int32 tensor)."""
        batch = lwe_in.shape[0]
        _check("rosetta_pbs_batch_multi_lut",
               load().rosetta_pbs_batch_multi_lut(self._h, _ptr(lwe_in), batch, _ptr(luts), luts.shape[0],
                                                  _ptr(lut_index), _ptr(lwe_out), _stream(stream)))
        return lwe_out

    def rosetta_blind_rotate_glwe_batch(self, lwe_in, glwe_in, glwe_out, stream=None):
        """Blind rotation of per-ciphertext GLWE test polynomials [batch][k+1][N]."""
        batch = lwe_in.shape[0]
        _check("rosetta_blind_rotate_glwe_batch",
               load().rosetta_blind_rotate_glwe_batch(self._h, _ptr(lwe_in), batch, _ptr(glwe_in), _ptr(glwe_out),
                                                      _stream(stream)))
        return glwe_out

    def rosetta_upload_trace_keys(self, keys, base_log, level, stream=None):
        n = keys.numel() if hasattr(keys, "numel") else keys.size
        _check("rosetta_upload_trace_keys",
               load().rosetta_upload_trace_keys(self._h, _ptr(keys), n, base_log, level, int(_is_device(keys)),
                                                _stream(stream)))

    def rosetta_trace_batch(self, glwe_in, glwe_out, stream=None):
        """RLWE trace of glwe_in [batch][2][N] (device) into glwe_out."""
        _check("rosetta_trace_batch", load().rosetta_trace_batch(self._h, _ptr(glwe_in), glwe_in.shape[0],
                                                                 _ptr(glwe_out), _stream(stream)))
        return glwe_out

    def rosetta_plaintext_mul_batch(self, glwe_in, plain_mul, glwe_out, plain_add=None, stream=None):
        """(P * A, P * B + Q) for glwe_in [batch][2][N] (device); plain_mul: host int64 [N]."""
        n = glwe_in.shape[-1]
        for name, v in (("plain_mul", plain_mul), ("plain_add", plain_add)):
            if v is not None and (v.shape != (n,) or v.dtype.itemsize != 8):
                raise ValueError(f"{name} must hold {n} 64-bit words")
        _check("rosetta_plaintext_mul_batch",
               load().rosetta_plaintext_mul_batch(self._h, _ptr(glwe_in), glwe_in.shape[0], _ptr(plain_mul),
                                                  None if plain_add is None else _ptr(plain_add), _ptr(glwe_out),
                                                  _stream(stream)))
        return glwe_out

    def rosetta_upload_lookup_table(self, p_hat, q_hat, a_hat, b_hat, stream=None):
        """Host tables of one segmented lookup: p_hat, q_hat [N]; a_hat, b_hat [n_seg][N]."""
        n = self.params.N
        n_seg = a_hat.shape[0]
        for name, v, shape in (("p_hat", p_hat, (n,)), ("q_hat", q_hat, (n,)), ("a_hat", a_hat, (n_seg, n)),
                               ("b_hat", b_hat, (n_seg, n))):
            if v.shape != shape or v.dtype.itemsize != 8:
                raise ValueError(f"{name} must be 64-bit words of shape {shape}")
        _check("rosetta_upload_lookup_table",
               load().rosetta_upload_lookup_table(self._h, n_seg, _ptr(p_hat), _ptr(q_hat), _ptr(a_hat), _ptr(b_hat),
                                                  _stream(stream)))

    def rosetta_segmented_lookup_batch(self, glwe_x, lwe_seg, glwe_out, stream=None):
        """Encrypted segmented lookup of each [[x]] (glwe_x [batch][2][N]) with segment index lwe_seg [batch][n+1]."""
        _check("rosetta_segmented_lookup_batch",
               load().rosetta_segmented_lookup_batch(self._h, _ptr(glwe_x), _ptr(lwe_seg), glwe_x.shape[0],
                                                     _ptr(glwe_out), _stream(stream)))
        return glwe_out

    def rosetta_selftest_wait_timeout(self, limit_us=10000, stream=None):
        """Make one bounded device wait expire (reported by sync_status as TIMEOUT)."""
        _check("rosetta_selftest_wait_timeout",
               load().rosetta_selftest_wait_timeout(self._h, limit_us, _stream(stream)))

    def rosetta_selftest_bounds(self, stream=None):
        """Make one bounds check of a ROSETTA_DEBUG build fail (reported by
        sync_status as BOUNDS); the regular build returns UNSUPPORTED_PARAMS."""
        _check("rosetta_selftest_bounds", load().rosetta_selftest_bounds(self._h, _stream(stream)))

    def rosetta_pbs_batch_noalloc(self, lwe_in, lut, lwe_out, stream=None):
        """rosetta_pbs_batch without any device allocation in the call (fixed
        in-library scratch; device buffers only, bounded batch)."""
        batch = lwe_in.shape[0]
        _check("rosetta_pbs_batch_noalloc", load().rosetta_pbs_batch_noalloc(self._h, _ptr(lwe_in), batch, _ptr(lut),
                                                                             _ptr(lwe_out), _stream(stream)))
        return lwe_out

    def rosetta_ntt_primes(self):
        """Primes of the blind rotation's exact external product: 3 or 4."""
        r = load().rosetta_ntt_primes(self._h)
        if r < 0:
            raise RosettaError("rosetta_ntt_primes", r)
        return r

    def rosetta_sync_status(self, stream=None):
        _check("rosetta_sync_status", load().rosetta_sync_status(self._h, _stream(stream)))

    # short aliases
    upload_bsk = rosetta_upload_bsk
    upload_ksk = rosetta_upload_ksk
    pbs_batch = rosetta_pbs_batch
    blind_rotate_extract_batch = rosetta_blind_rotate_extract_batch
    keyswitch_batch = rosetta_keyswitch_batch
    pbs_batch_multi_lut = rosetta_pbs_batch_multi_lut
    blind_rotate_glwe_batch = rosetta_blind_rotate_glwe_batch
    upload_trace_keys = rosetta_upload_trace_keys
    trace_batch = rosetta_trace_batch
    plaintext_mul_batch = rosetta_plaintext_mul_batch
    upload_lookup_table = rosetta_upload_lookup_table
    segmented_lookup_batch = rosetta_segmented_lookup_batch
    selftest_wait_timeout = rosetta_selftest_wait_timeout
    selftest_bounds = rosetta_selftest_bounds
    ntt_primes = rosetta_ntt_primes
    sync_status = rosetta_sync_status
