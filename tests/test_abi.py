"""The C ABI library loads and exports every entry point include/agnes.h
declares (no GPU needed; no compute is launched)."""
import ctypes
import os
import re

import pytest

from paper_2601_01473_gb300 import agnes

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            text = open(os.path.join(ROOT, "include", f)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(agnes_[a-z0-9_]+)\s*\(", text))
    return names


@pytest.fixture(scope="module")
def L():
    from paper_2601_01473_gb300 import build
    build.build()
    return agnes.lib()


def test_every_declared_symbol_is_exported(L):
    names = _declared()
    assert "agnes_load_graph" in names and "agnes_prepare_hyperbatch" in names
    for n in names:
        assert hasattr(L, n), n


def test_binding_covers_the_header(L):
    assert _declared() <= set(agnes.SIGNATURES)


def test_null_arguments_are_rejected_without_a_device(L):
    ctx = ctypes.c_void_p()
    assert L.agnes_load_graph(None, 0, None, ctypes.byref(ctx)) == 1
    assert ctx.value is None
    assert b"desc" in L.agnes_last_error(None)
    fan = (ctypes.c_int32 * 1)(5)
    assert L.agnes_prepare_hyperbatch(None, None, 1, 1, fan, 1, 0, 0, None) == 1
    assert L.agnes_fetch_minibatch(None, 0, None) == 1
    assert L.agnes_set_launch_mode(None, 1) == 1
    assert L.agnes_free(None) == 0


def test_status_strings(L):
    for code in range(8):
        assert L.agnes_status_string(code)
    assert L.agnes_status_string(0) == b"ok"


def test_bad_descs_fail_before_any_cuda_call(L):
    d = agnes._GraphDesc()
    d.num_nodes = 0
    ctx = ctypes.c_void_p()
    assert L.agnes_load_graph(ctypes.byref(d), 0, None, ctypes.byref(ctx)) == 1
    d.num_nodes = 10
    d.offsets_bits = 16
    assert L.agnes_load_graph(ctypes.byref(d), 0, None, ctypes.byref(ctx)) == 1
    d.num_nodes = 1 << 31
    d.offsets_bits = 64
    assert L.agnes_load_graph(ctypes.byref(d), 0, None, ctypes.byref(ctx)) == 2
