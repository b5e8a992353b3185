"""CPU checks of the boundary: the shared library builds, loads, and exports
every entry point include/tv.h declares (no GPU needed, no compute calls)."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    src = open(os.path.join(ROOT, "include", "tv.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tv_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_2505_12398_gb300.build import build
    path = build()
    return ctypes.CDLL(path)


def test_header_declares_the_boundary():
    names = declared_functions()
    for need in ("tv_create", "tv_verify_batch", "tv_destroy"):
        assert need in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_error_strings_and_version(lib):
    lib.tv_strerror.restype = ctypes.c_char_p
    for code in (0, -1, -2, -3, -4, -5, -6):
        assert lib.tv_strerror(code) and lib.tv_strerror(code) != b"unknown error code"
    assert lib.tv_strerror(-99) == b"unknown error code"
    assert lib.tv_version() >= 100


def test_binding_signatures_cover_the_header():
    from paper_2505_12398_gb300._binding import _SIGS
    assert set(_SIGS) == set(declared_functions())


def test_product_path_does_not_import_the_oracle():
    pkg = os.path.join(ROOT, "paper_2505_12398_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in text and "from oracle" not in text, f


def _cuda_lib_dir():
    for d in ("/usr/local/cuda/lib64", "/usr/local/cuda/targets/sbsa-linux/lib",
              "/usr/local/cuda/targets/x86_64-linux/lib"):
        if os.path.exists(os.path.join(d, "libcudart.so")):
            return d
    return None


def test_header_is_plain_c_and_links(lib, tmp_path):
    """include/tv.h compiles as strict C99 and as C++, and a C program that
    takes every entry point's address links against libtv.so and runs the
    host-side checks (no device needed)."""
    import shutil
    import subprocess
    cc, cxx = shutil.which("gcc"), shutil.which("g++")
    cudadir = _cuda_lib_dir()
    if not cc or not cxx or not cudadir:
        pytest.skip("no C toolchain or CUDA runtime library")
    inc = os.path.join(ROOT, "include")
    src = os.path.join(ROOT, "tests", "c_abi", "use_abi.c")
    libdir = os.path.dirname(lib._name)
    exe = str(tmp_path / "use_abi")
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-I", inc,
                        src, "-o", exe, "-L", libdir, "-ltv", f"-Wl,-rpath,{libdir}",
                        f"-Wl,-rpath-link,{cudadir}", f"-Wl,-rpath,{cudadir}"],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    hdr = tmp_path / "hdr.cc"
    hdr.write_text('#include "tv.h"\nint main() { return tv_version() > 0 ? 0 : 1; }\n')
    r = subprocess.run([cxx, "-std=c++17", "-Wall", "-Werror", "-fsyntax-only", "-I", inc,
                        str(hdr)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), (r.returncode, r.stdout,
                                                                   r.stderr)


def test_binding_checks_output_tensors():
    """Outputs the kernels write are checked for dtype, shape, contiguity and
    device before any call (the kernels trust the sizes)."""
    import torch
    from paper_2505_12398_gb300._binding import _check_out
    cpu = torch.device("cpu")
    _check_out(torch.zeros(2, 3, dtype=torch.int32), torch.int32, (2, 3), cpu)
    for bad in (torch.zeros(2, 3), torch.zeros(3, 2, dtype=torch.int32),
                torch.zeros(3, 2, dtype=torch.int32).t()):
        with pytest.raises(ValueError):
            _check_out(bad, torch.int32, (2, 3), cpu)


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """Without the compiled library the binding raises; there is no CPU
    implementation to fall back to."""
    from paper_2505_12398_gb300 import _binding
    monkeypatch.setattr(_binding, "_LIB", None)
    monkeypatch.setattr(_binding, "library_path", lambda: str(tmp_path / "libtv.so"))
    with pytest.raises(ImportError):
        _binding.library()
    with pytest.raises(ImportError):
        _binding.Verifier(1000, 7, 4, "bf16")
