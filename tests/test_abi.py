"""The C-ABI library builds, loads without a GPU and exports every entry point
that include/kvm.h declares.  Only argument validation that returns before any
CUDA call is exercised here."""
import ctypes as C
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "kvm.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2609_18935_gb300 import build_lib, kvm
    if not os.path.exists(kvm.LIB_PATH):
        build_lib.build()
    return kvm.load_library()


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*[A-Za-z_][\w \*]*?\b(kvm_\w+)\s*\(", text, flags=re.M)))


def test_header_declares_the_hot_path():
    names = _declared()
    for n in ["kvm_kv_compact", "kvm_tail_attn_prefill", "kvm_gdn_chunk_scan_from_state",
              "kvm_update_round", "kvm_create", "kvm_destroy"]:
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2609_18935_gb300 import kvm
    out = subprocess.run(["nm", "-D", "--defined-only", kvm.LIB_PATH], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (kvm_\w+)$", out, flags=re.M))
    missing = [n for n in _declared() if n not in exported]
    assert not missing, missing
    for n in _declared():
        getattr(lib, n)


def test_binding_signatures_cover_header(lib):
    from paper_2609_18935_gb300 import kvm
    assert set(_declared()) == set(kvm._SIGS)


def _desc(kvm, kinds, **kw):
    arr = (C.c_int32 * len(kinds))(*kinds)
    d = dict(n_q_heads=16, n_kv_heads=2, head_dim=256, rotary_dim=64, rope_theta=1e4,
             n_gdn_heads=16, d_k=128, d_v=128)
    d.update(kw)
    return kvm.ModelDesc(len(kinds), arr, d["n_q_heads"], d["n_kv_heads"], d["head_dim"], d["rotary_dim"],
                         d["rope_theta"], d["n_gdn_heads"], d["d_k"], d["d_v"], d.get("conv_kernel", 0)), arr


@pytest.mark.parametrize("kw,code", [({"head_dim": 96}, 6), ({"n_q_heads": 12, "n_kv_heads": 5}, 6),
                                     ({"n_q_heads": 24, "n_kv_heads": 2}, 6), ({"rotary_dim": 63}, 6),
                                     ({"d_k": 96}, 6), ({"d_v": 40}, 6), ({"d_v": 160}, 6),
                                     ({"rope_theta": -1.0}, 1), ({"conv_kernel": 3}, 6)])
def test_create_rejects_unsupported_shapes(lib, kw, code):
    from paper_2609_18935_gb300 import kvm
    desc, keep = _desc(kvm, [0, 0, 0, 1], **kw)
    caps = (C.c_int32 * 1)(1024)
    h = C.c_void_p()
    assert lib.kvm_create(C.byref(desc), 1, caps, 256, C.byref(h)) == code
    assert lib.kvm_last_error().decode()
    assert not h.value


def test_create_rejects_bad_population(lib):
    from paper_2609_18935_gb300 import kvm
    desc, keep = _desc(kvm, [0, 1])
    h = C.c_void_p()
    caps = (C.c_int32 * 2)(1024, 0)
    assert lib.kvm_create(C.byref(desc), 2, caps, 256, C.byref(h)) == kvm.KVM_E_INVAL
    assert lib.kvm_create(C.byref(desc), 0, caps, 256, C.byref(h)) == kvm.KVM_E_INVAL
    assert lib.kvm_create(C.byref(desc), 1, caps, 0, C.byref(h)) == kvm.KVM_E_INVAL
    assert lib.kvm_create(None, 1, caps, 16, C.byref(h)) == kvm.KVM_E_INVAL


def test_null_context_is_rejected(lib):
    from paper_2609_18935_gb300 import kvm
    assert lib.kvm_advance(None, None) == kvm.KVM_E_INVAL
    assert lib.kvm_check(None, None) == kvm.KVM_E_INVAL
    assert lib.kvm_launch_count(None) == 0


def test_debug_build_exports_the_same_symbols():
    """The canary-checking build (-DKVM_DEBUG) compiles and exports the same
    C ABI as the release library."""
    from paper_2609_18935_gb300 import build_lib
    path = build_lib.build(debug=True)
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (kvm_\w+)$", out, flags=re.M))
    assert set(_declared()) <= exported
