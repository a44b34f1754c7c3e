"""The C-ABI library builds for sm_103a, loads, and exports every entry point
declared in include/oos.h (host-only checks, except the one gpu-marked test of
config validation, which needs the device's SM count)."""

import ctypes
import os
import re

import pytest

from paper_2608_00814_gb300 import _build
from paper_2608_00814_gb300 import binding as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared():
    with open(os.path.join(ROOT, "include", "oos.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(oos_\w+)\s*\(", text)))


def test_every_declared_symbol_is_exported():
    _build.build()
    lib = ctypes.CDLL(_build.LIB)
    names = declared()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings_and_config_rejection():
    _build.build()
    L = B.lib()
    for code in (B.OOS_OK, B.OOS_EINVAL, B.OOS_ECAPACITY, B.OOS_ECUDA, B.OOS_ETREE, B.OOS_ETIMEOUT,
                 B.OOS_EUNSUPPORTED, B.OOS_EWORKSPACE):
        assert B.oos_status_string(code) != "unknown status"
    bad = B.OosModelConfig(0, 256, 4, 2, 64, 512, 1024, 0, 0, 0, 1e-6, 1e6, 8, 0)   # zero layers
    assert L.oos_workspace_bytes(ctypes.byref(bad)) == 0
    bad = B.OosModelConfig(2, 256, 4, 3, 64, 512, 1024, 0, 0, 0, 1e-6, 1e6, 8, 0)   # nq % nkv != 0
    assert L.oos_workspace_bytes(ctypes.byref(bad)) == 0
    bad = B.OosModelConfig(2, 256, 4, 2, 64, 512, 1024, 0, 0, 0, 1e-6, 1e6, 129, 0)  # max_T > 128
    assert L.oos_workspace_bytes(ctypes.byref(bad)) == 0
    h = ctypes.c_void_p()
    assert L.oos_model_create(None, None, None, 0, ctypes.byref(h)) == B.OOS_EINVAL
    assert L.oos_model_destroy(None) == B.OOS_EINVAL
    assert L.oos_accept_walk(None, None, None, 4, None, None, None, None, None, None) == B.OOS_EINVAL


def test_library_is_sm103a_only():
    flags = _build._flags()
    assert "arch=compute_103a,code=sm_103a" in " ".join(flags)


@pytest.mark.gpu
def test_rope_rescaling_config_validation():
    """Llama-3.1 rotary rescaling fields: accepted with hi > lo > 0 and L >= 1,
    rejected otherwise (workspace size 0).  Needs a device: the workspace size
    depends on its SM count."""
    _build.build()
    L = B.lib()
    good = B.OosModelConfig(2, 256, 4, 2, 64, 512, 1024, 0, 0, 0, 1e-6, 5e5, 8, 0, 8.0, 1.0, 4.0, 8192)
    assert L.oos_workspace_bytes(ctypes.byref(good)) > 0
    plain = B.OosModelConfig(2, 256, 4, 2, 64, 512, 1024, 0, 0, 0, 1e-6, 5e5, 8, 0, 0.0, 0.0, 0.0, 0)
    assert L.oos_workspace_bytes(ctypes.byref(plain)) > 0      # factor 0: the other fields are ignored
    for lo, hi, orig in ((4.0, 4.0, 8192), (0.0, 4.0, 8192), (1.0, 4.0, 0)):
        bad = B.OosModelConfig(2, 256, 4, 2, 64, 512, 1024, 0, 0, 0, 1e-6, 5e5, 8, 0, 8.0, lo, hi, orig)
        assert L.oos_workspace_bytes(ctypes.byref(bad)) == 0
    bad = B.OosModelConfig(2, 256, 4, 2, 64, 512, 1024, 0, 0, 0, 1e-6, 5e5, 8, 0, float("nan"), 1.0, 4.0, 8192)
    assert L.oos_workspace_bytes(ctypes.byref(bad)) == 0
