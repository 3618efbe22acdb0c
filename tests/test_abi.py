"""CPU checks of the C ABI: the library builds for sm_103a, loads, and exports
every entry point the public header declares (no compute without a GPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "cacheroute.h")


def _declared():
    src = open(HEADER).read()
    return sorted(set(re.findall(r"^CR_API [^(]*?\b(cr_[a-z_]+)\(", src, flags=re.M)))


@pytest.fixture(scope="module")
def built():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_19677_gb300 as P
    return P


def test_header_declares_the_four_path_calls():
    d = _declared()
    for name in ("cr_hash_prefixes", "cr_build_plan", "cr_route_batch", "cr_shadow_replay"):
        assert name in d


def test_library_exports_every_declared_symbol(built):
    P = built
    lib = ctypes.CDLL(P.LIB_PATH)
    missing = [s for s in _declared() if not hasattr(lib, s)]
    assert not missing, missing
    assert sorted(P.EXPORTS) == _declared()


def test_binding_loads_and_reports_errors_without_device(built):
    P = built
    L = P.lib()
    # cr_create on a machine without a usable device fails cleanly with a message
    h = ctypes.c_void_p()
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    st = L.cr_create(ctypes.byref(h), 0, None)
    assert st != 0
    assert len(L.cr_last_error(None)) > 0
    assert L.cr_launch_count(None) == 0


def test_product_never_imports_the_oracle():
    pkg = os.path.join(ROOT, "paper_2608_19677_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                txt = open(os.path.join(dirpath, f)).read()
                assert not re.search(r"^\s*(import|from)\s+oracle\b", txt, flags=re.M), f
                assert "cr_oracle" not in txt and "libcr_oracle" not in txt, f


def test_debug_build_compiles_and_exports_every_symbol():
    # the bounds-checking variant (-DCR_DEBUG_CHECKS) builds for sm_103a and exports the same ABI
    from paper_2608_19677_gb300 import buildlib
    path = buildlib.build(debug=True)
    assert path.endswith("libcacheroute_debug.so") and os.path.exists(path)
    lib = ctypes.CDLL(path)
    missing = [s for s in _declared() if not hasattr(lib, s)]
    assert not missing, missing
