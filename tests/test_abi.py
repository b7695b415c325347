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
    assert aio.aio_abi_version() == aio.AIO_ABI_VERSION == 8
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


def test_new_entry_points_reject_bad_arguments_before_cuda(aio):
    """The chained step, attention, PLD and routing entry points check their arguments on the host
    and return before any CUDA call (these run without a GPU)."""
    lib = aio.lib()
    bad = aio.AIO_ERR_INVALID_ARG
    assert lib.aio_decode_step_create_chained(None, None, None, 0, 1, 0) == bad
    # attention: NULL pointers, then head_dim, M and L ranges, q_stride, alignment
    assert lib.aio_attention_decode(None, 128, None, None, 1, 128, 16, 16, 1, None, None, 0, None) == bad
    p = 1 << 20   # any non-NULL address: nothing is dereferenced before the checks below fail
    assert lib.aio_attention_decode(p, 128, p, p, 1, 64, 16, 16, 1, p, p, 0, None) == aio.AIO_ERR_UNSUPPORTED
    assert lib.aio_attention_decode(p, 128, p, p, 1, 128, 16, 16, 9, p, p, 0, None) == bad
    assert lib.aio_attention_decode(p, 128, p, p, 1, 128, 16, 17, 1, p, p, 0, None) == bad
    assert lib.aio_attention_decode(p, 64, p, p, 1, 128, 16, 16, 1, p, p, 0, None) == bad
    assert lib.aio_attention_decode(p + 4, 128, p, p, 1, 128, 16, 16, 1, p, p, 0, None) == aio.AIO_ERR_ALIGNMENT
    assert lib.aio_attention_workspace_bytes(9, None) == bad
    # prompt lookup and routing
    assert lib.aio_pld_draft(None, 10, 6, 2, None, None) == bad
    assert lib.aio_pld_draft(p, 0, 6, 2, p, None) == bad
    assert lib.aio_pld_draft(p, 10, 6, 8, p, None) == bad
    assert lib.aio_pld_draft(p + 2, 10, 6, 2, p, None) == aio.AIO_ERR_ALIGNMENT
    assert lib.aio_argmax_rows(p, 1, 10, 9, p, None) == bad
    assert lib.aio_pld_accept(None, p, p, None) == bad
    assert lib.aio_route(p, p, 0, 0, 10, ctypes.c_float(0.45), p, None) == bad
    assert lib.aio_route(p, p, 3, 3, 10, ctypes.c_float(0.45), p, None) == bad
    assert lib.aio_route(p, p, 3, 0, -1, ctypes.c_float(0.45), p, None) == bad
    assert lib.aio_route(p, p, 3, 0, 10, ctypes.c_float(float("nan")), p, None) == bad
