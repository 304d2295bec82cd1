"""The C ABI library loads, exports every entry point include/osprey.h declares,
and rejects bad host-visible arguments before touching the GPU (no compute
calls here: these run without a GPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__ as g
    g.build()
    return ctypes.CDLL(os.path.join(ROOT, "paper_2609_09338_gb300", "libosprey.so"))


def _declared():
    hdr = open(os.path.join(ROOT, "include", "osprey.h")).read()
    hdr = re.sub(r"/\*.*?\*/", "", hdr, flags=re.S)
    return sorted(set(re.findall(r"\b(osprey_[a-z_0-9]+)\s*\(", hdr)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert "osprey_draft_step" in names and "osprey_verify" in names and "osprey_kv_append" in names
    for n in names:
        assert hasattr(lib, n), n


def test_binding_covers_the_header(lib):
    from paper_2609_09338_gb300 import binding
    assert sorted(binding.EXPORTED) == _declared()


def test_verify_rejects_bad_arguments_on_host(lib):
    from paper_2609_09338_gb300 import binding as ob
    f = ob._c_verify
    buf = ctypes.create_string_buffer(1 << 16)
    p = ctypes.cast(buf, ctypes.c_void_p)
    # K = 0 -> INVALID_ARG before any launch
    assert f(1, 0, 16, 0, p, p, p, 1.0, p, p, p, p, p, None, p, 1 << 16, None, None) == -1
    assert "K in 1..15" in ob.osprey_last_error()
    # unknown dtype -> DTYPE
    assert f(1, 2, 16, 7, p, p, p, 1.0, p, p, p, p, p, None, p, 1 << 16, None, None) == -3
    # sampled mode without draft logits -> INVALID_ARG
    assert f(1, 2, 16, 0, p, None, p, 1.0, p, p, p, p, p, None, p, 1 << 16, None, None) == -1
    # negative temperature -> INVALID_ARG
    assert f(1, 2, 16, 0, p, p, p, -1.0, p, p, p, p, p, None, p, 1 << 16, None, None) == -1
    # workspace too small -> CAPACITY
    need = ob.osprey_verify_workspace_bytes(4, 3, 5000)
    assert need > 0
    assert f(4, 3, 5000, 0, p, p, p, 1.0, p, p, p, p, p, None, p, need - 1, None, None) == -4
    # B = 0 is an empty call
    assert f(0, 3, 16, 0, None, None, None, 1.0, None, None, None, None, None, None, None, 0, None, None) == 0
    assert ob.osprey_verify_workspace_bytes(1, 0, 16) == 0


def test_create_validates_shape_before_the_device(lib):
    from paper_2609_09338_gb300 import binding as ob
    cfg = ob.osprey_config(256, 1, 4, 2, 96, 768, 4096, 1536, 16, 1e-6, 1e6)   # head_dim 96
    w = ob.osprey_weights()
    h = ctypes.c_void_p()
    assert ob._c_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)) == -2
    assert "head_dim" in ob.osprey_last_error()
    cfg = ob.osprey_config(256, 1, 4, 2, 64, 768, 4096, 1536, 8, 1e-6, 1e6)    # page 8
    assert ob._c_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)) == -2
    cfg = ob.osprey_config(256, 1, 4, 2, 64, 768, 4096, 1536, 16, 1e-6, 1e6)   # null weights
    assert ob._c_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)) == -1
    assert ob._c_create(None, ctypes.byref(w), ctypes.byref(h)) == -1


def test_kv_append_and_draft_reject_null_pointers(lib):
    from paper_2609_09338_gb300 import binding as ob
    kv = ob.osprey_kv()
    assert ob._c_kv_append(None, ctypes.byref(kv), 1, None, 0, None, None, None, None) == -1
    assert ob._c_draft(None, ctypes.byref(kv), 1, 1, 1, None, None, None, 1.0, None, None, None, None, None,
                       None, 0, None, None) == -1


def test_selftest_wait_timeout_validates_on_host(lib):
    from paper_2609_09338_gb300 import binding as ob
    f = ob._c_selftest_wait
    assert f(0, ctypes.c_void_p(16), None) == -1               # INVALID_ARG, before any launch
    assert f(3_000_000_000, ctypes.c_void_p(16), None) == -1
    assert f(1000, None, None) == -1
    assert "limit_cycles" in ob.osprey_last_error()


def test_logits_free_entry_points_validate_on_host(lib):
    from paper_2609_09338_gb300 import binding as ob
    kv = ob.osprey_kv()
    p = ctypes.c_void_p(256)
    # draft_step_hidden without the hidden buffer, and with a null context
    assert ob._c_draft_hidden(p, ctypes.byref(kv), 1, 1, 1, p, p, p, 1.0, p, p, p, p, None, p, 1 << 20, None,
                              None) == -1
    assert "draft_hidden" in ob.osprey_last_error()
    assert ob._c_draft_hidden(None, ctypes.byref(kv), 1, 1, 1, p, p, p, 1.0, p, p, p, p, p, p, 1 << 20, None,
                              None) == -1
    # verify_hidden: null context; no workspace size without a context
    f = ob._c_verify_hidden
    assert f(None, 1, 2, 0, p, p, p, p, p, 1.0, p, p, p, p, p, None, p, 1 << 20, None, None) == -1
    assert ob._c_verify_hidden_ws(None, 1, 2) == 0


def test_status_names_cover_bounds_checked_builds(lib):
    from paper_2609_09338_gb300 import binding as ob
    assert ob.status_name(0) == "OK" and ob.status_name(-6) == "TIMEOUT"
    assert ob.status_name(-1342) == "BOUNDS(line 342)"
    assert ob.status_name(-77).startswith("UNKNOWN")
