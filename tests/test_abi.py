"""The C-ABI library builds, loads and exports every entry point include/tss.h declares (no GPU:
no compute call is made)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    with open(os.path.join(ROOT, "include", "tss.h")) as f:
        src = f.read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tss_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def libtss():
    from paper_2609_26100_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_the_boundary():
    names = _declared()
    for must in ("tss_create", "tss_set_skip_config", "tss_verify", "tss_destroy"):
        assert must in names


def test_library_exports_every_declared_symbol(libtss):
    missing = [n for n in _declared() if not hasattr(libtss, n)]
    assert missing == []


def test_binding_covers_the_exports(libtss):
    from paper_2609_26100_gb300 import native
    assert sorted(native.EXPORTS) == _declared()


def test_status_strings_without_gpu(libtss):
    libtss.tss_status_string.restype = ctypes.c_char_p
    assert libtss.tss_status_string(0) == b"ok"
    assert libtss.tss_status_string(3) == b"KV cache capacity exceeded"


def test_library_built_for_sm103a_only():
    from paper_2609_26100_gb300 import build
    assert build.ARCH == ("-gencode", "arch=compute_103a,code=sm_103a")
