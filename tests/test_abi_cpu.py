"""The C ABI library on a machine without a GPU: it builds, loads, exports every entry point that
include/clearmoe.h declares, and rejects bad descriptors on the host before touching CUDA."""
import ctypes
import pathlib
import re

import pytest

from paper_2606_28516_gb300 import build as B
from paper_2606_28516_gb300 import clearmoe as cm

HEADER = pathlib.Path(__file__).resolve().parents[1] / "include"


def declared_entry_points():
    names = set()
    for h in HEADER.glob("*.h"):
        text = re.sub(r"/\*.*?\*/", "", h.read_text(), flags=re.S)
        names |= set(re.findall(r"^[A-Za-z_][\w \*]*?\b(clearmoe_\w+)\s*\(", text, flags=re.M))
    return sorted(names)


@pytest.fixture(scope="module")
def lib():
    B.build()
    return cm.lib()


def test_header_declares_the_abi():
    names = declared_entry_points()
    for n in ("clearmoe_layer_create", "clearmoe_ffn_forward", "clearmoe_dense_ffn_forward",
              "clearmoe_route", "clearmoe_get_routing", "clearmoe_layer_status"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    for n in declared_entry_points():
        assert hasattr(lib, n), n
        assert n in cm._SIGS, f"binding lacks {n}"


def test_strerror_and_version(lib):
    assert cm.clearmoe_strerror(cm.ETIMEOUT) == "a bounded device-side wait timed out"
    assert cm.clearmoe_strerror(12345) == "unknown status"
    assert cm.clearmoe_version() >= 100


def test_bad_descriptors_rejected_on_host(lib):
    h = ctypes.c_void_p()
    assert lib.clearmoe_layer_create(None, ctypes.byref(h)) == cm.EINVAL
    for kw, code in ((dict(max_tokens=0), cm.EINVAL), (dict(dtype=7), cm.EINVAL),
                     (dict(max_E=17), cm.EUNSUPPORTED), (dict(max_r=512), cm.EUNSUPPORTED),
                     (dict(d=100), cm.EUNSUPPORTED)):
        args = dict(max_tokens=100, d=128, hidden=512, max_E=4, max_r=32, dtype=cm.BF16) | kw
        desc = cm.clearmoe_layer_desc(**args)
        assert lib.clearmoe_layer_create(ctypes.byref(desc), ctypes.byref(h)) == code, kw
    assert lib.clearmoe_layer_destroy(None) == cm.OK
    assert lib.clearmoe_layer_status(None) == cm.EINVAL
    assert lib.clearmoe_route(None, None, 1, None, 1, None) == cm.EINVAL
