"""CPU tests of the boundary: the library loads and exports every symbol the
header declares, and host-side argument checks reject bad calls before any
device work (these paths return before touching a GPU)."""
import ctypes
import os
import re

import pytest

from paper_2606_19528_gb300 import lora, build

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "lora.h")


def _declared():
    src = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:int|int64_t|const char\*)\s+(lora_\w+)\s*\(", src, re.M)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(lora._LIB_PATH):
        build.build_cuda()
    return lora.library()


def test_header_declares_the_binding_names():
    assert _declared() == sorted(lora.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_strerror_and_version(lib):
    assert lora.lora_version() >= 100
    for code in (lora.LORA_OK, lora.LORA_EINVAL, lora.LORA_ENULL, lora.LORA_EALIGN, lora.LORA_ECUDA,
                 lora.LORA_ETIMEOUT, lora.LORA_EWORKSPACE, lora.LORA_EDEVICE):
        assert lora.lora_strerror(code)
    assert lora.lora_strerror(12345) == "unknown error"


def test_null_arguments_are_rejected(lib):
    n = ctypes.c_size_t(0)
    assert lib.lora_workspace_size(None, 1, ctypes.byref(n)) == lora.LORA_ENULL
    assert lib.lora_linear_fwd(None, None, None, None, None, None, None, None, 0, None) == lora.LORA_ENULL
    assert lib.lora_stack_step(None, 1, 1, None, 0, None) == lora.LORA_ENULL
    st = lora.make_shape(128, 256, 256, 8, 2.0)
    assert lib.lora_stack_step(ctypes.byref(lora.make_proj(st)), 0, 1, None, 0, None) == lora.LORA_EINVAL
    assert lib.lora_stack_step(ctypes.byref(lora.make_proj(st)), 1, 7, None, 0, None) == lora.LORA_EINVAL
