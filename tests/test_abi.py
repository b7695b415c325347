"""The C ABI library loads, exports every symbol include/aio.h declares, and rejects bad
arguments on the host before touching CUDA (CPU only, no compute calls)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "aio.h")


@pytest.fixture(scope="module")
def aio():
    from paper_2604_09752_gb300 import build
    build.build()
    from paper_2604_09752_gb300 import aio as mod
    return mod


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b(aio_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ["aio_linear_create", "aio_linear_run", "aio_linear_pack", "aio_linear_destroy",
                     "aio_decode_step_create", "aio_decode_step", "aio_decode_step_destroy",
                     "aio_status_string", "aio_last_error"]:
        assert required in names


def test_library_exports_every_declared_symbol(aio):
    lib = ctypes.CDLL(aio.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_no_torch_types_in_signatures():
    text = open(HEADER).read()
    assert "torch" not in text.lower().replace("(pytorch)", "")
    assert "at::" not in text and "Tensor" not in text


def test_abi_version_and_status_strings(aio):
    assert aio.aio_abi_version() == 5
    for code in range(8):
        assert aio.aio_status_string(code).startswith("AIO_")
    assert aio.aio_status_string(99) == "AIO_ERR_UNKNOWN"


@pytest.mark.parametrize("K,N,wt,max_M,flags", [
    (15, 8, 0, 1, 0),          # K not a multiple of 16
    (0, 8, 0, 1, 0),
    (16, 0, 0, 1, 0),          # N < 1
    (16, 8, 2, 1, 0),          # unknown weight type
    (16, 8, 0, 0, 0),          # max_M < 1
    (16, 8, 0, 9, 0),          # max_M > 8
    (16, 8, 0, 1, 0x80),       # unknown flag
    ((1 << 20) + 16, 8, 0, 1, 0),
])
def test_create_rejects_bad_arguments_before_cuda(aio, K, N, wt, max_M, flags):
    with pytest.raises(aio.AioError) as e:
        aio.aio_linear_create(K, N, wt, max_M, flags)
    assert e.value.status == aio.AIO_ERR_INVALID_ARG


def test_null_handles_rejected(aio):
    lib = aio.lib()
    assert lib.aio_linear_run(None, None, 1, 16, 16, None, None, None, None) == aio.AIO_ERR_INVALID_ARG
    assert lib.aio_decode_step(None, None) == aio.AIO_ERR_INVALID_ARG
    assert lib.aio_linear_destroy(None) == aio.AIO_OK
    assert lib.aio_decode_step_destroy(None) == aio.AIO_OK
    assert lib.aio_decode_step_create(None, None, 0, 1, 0) == aio.AIO_ERR_INVALID_ARG
    assert lib.aio_probe_read(None, 4096, None, None) == aio.AIO_ERR_INVALID_ARG
    assert b"NULL" in lib.aio_last_error() or b"null" in lib.aio_last_error()


def test_binding_fails_loudly_without_library(tmp_path):
    # the binding never falls back: with libaio.so absent, importing it raises
    import subprocess, sys, shutil
    pkg = tmp_path / "paper_2604_09752_gb300"
    shutil.copytree(os.path.join(ROOT, "paper_2604_09752_gb300"), pkg,
                    ignore=shutil.ignore_patterns("*.so", "_build", "__pycache__"))
    shutil.copytree(os.path.join(ROOT, "include"), tmp_path / "include")
    r = subprocess.run([sys.executable, "-c", "import paper_2604_09752_gb300.aio"], cwd=tmp_path,
                       capture_output=True, text=True)
    assert r.returncode != 0 and "libaio.so is missing" in r.stderr
