"""The C-ABI library builds, loads and exports every function include/rosetta.h
declares; argument checks that happen before any CUDA call behave as
documented.  No test here touches a GPU."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "rosetta.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(rosetta_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    import shutil
    if not (shutil.which("nvcc") or os.path.exists("/usr/local/cuda/bin/nvcc")):
        pytest.skip("nvcc not available")
    from paper_2609_16915_gb300 import build
    build.build()
    import paper_2609_16915_gb300 as R
    return R.load()


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ["rosetta_params_init", "rosetta_upload_bsk", "rosetta_upload_ksk", "rosetta_pbs_batch",
                 "rosetta_keyswitch_batch", "rosetta_blind_rotate_extract_batch", "rosetta_sync_status",
                 "rosetta_destroy", "rosetta_status_string"]:
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_binding_exposes_every_declared_symbol():
    import paper_2609_16915_gb300 as R
    assert set(declared_functions()) <= set(R.EXPORTS)


def test_status_strings(lib):
    import paper_2609_16915_gb300 as R
    for code, text in R.STATUS.items():
        assert R.rosetta_status_string(code) == text


def test_argument_checks_before_cuda(lib):
    import paper_2609_16915_gb300 as R
    h = ctypes.c_void_p()
    assert lib.rosetta_params_init(None, None, 0) == -1
    assert lib.rosetta_params_init(ctypes.byref(h), None, 0) == -1
    base = dict(lwe_dim=64, glwe_dim=1, poly_size=256, pbs_base_log=10, pbs_level=2, ks_base_log=4, ks_level=4,
                msg_bits=3, max_batch=0)
    for bad in [dict(poly_size=300), dict(poly_size=16384), dict(glwe_dim=2), dict(pbs_base_log=0),
                dict(pbs_base_log=29), dict(pbs_base_log=20, pbs_level=4), dict(ks_base_log=17),
                dict(msg_bits=8), dict(lwe_dim=0)]:
        prm = R.rosetta_params(**{**base, **bad})
        assert lib.rosetta_params_init(ctypes.byref(h), ctypes.byref(prm), 0) == -2, bad
        assert h.value is None
    # null contexts
    assert lib.rosetta_pbs_batch(None, None, 0, None, None, None) == -1
    assert lib.rosetta_keyswitch_batch(None, None, 0, None, None) == -1
    assert lib.rosetta_sync_status(None, None) == -1
    lib.rosetta_destroy(None)


def build_c_client(out_path):
    """Compile tests/c_abi_demo.c, a plain C99 program that uses the library
    through include/rosetta.h alone, and link it against librosetta.so."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not installed")
    here = os.path.dirname(os.path.abspath(__file__))
    root = os.path.dirname(here)
    pkg = os.path.join(root, "paper_2609_16915_gb300")
    cmd = [gcc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(root, "include"),
           os.path.join(here, "c_abi_demo.c"), "-L", pkg, "-lrosetta", f"-Wl,-rpath,{pkg}",
           "-L/usr/local/cuda/lib64", "-o", out_path]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return out_path


def test_c_client_compiles_and_links(lib, tmp_path):
    """The header is plain C and the library links from C without CUDA headers."""
    assert os.path.exists(build_c_client(str(tmp_path / "c_abi_demo")))


def declared_arity():
    """Parameter count of every prototype in the header."""
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    out = {}
    for name, params in re.findall(r"\b(rosetta_[a-z_]+)\s*\(([^)]*)\)\s*;", text):
        params = params.strip()
        out[name] = 0 if params in ("", "void") else params.count(",") + 1
    return out


def test_binding_argument_counts_match_the_header(lib):
    arity = declared_arity()
    assert set(arity) == set(declared_functions())
    for name, n in arity.items():
        assert len(getattr(lib, name).argtypes) == n, name


def test_debug_build_compiles_and_exports_the_same_symbols(lib):
    """The ROSETTA_DEBUG library (device-side bounds checks) builds from the
    same sources and has the same boundary."""
    from paper_2609_16915_gb300 import build
    path = build.build(debug=True)
    dbg = ctypes.CDLL(path)
    for name in declared_functions():
        assert hasattr(dbg, name), name
    dbg.rosetta_status_string.restype = ctypes.c_char_p
    assert dbg.rosetta_status_string(-7) == b"device-side bounds check failed (debug build)"
