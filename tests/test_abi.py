"""The C-ABI library builds, loads and exports every function include/lca.h declares (CPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = []
    for f in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if not f.endswith(".h"):
            continue
        text = open(os.path.join(ROOT, "include", f)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names += re.findall(r"^\s*(?:int|size_t|const char\s*\*)\s+(lca_\w+)\s*\(", text, flags=re.M)
    return names


def test_header_declares_the_step_api():
    names = declared_functions()
    for n in ("lca_create", "lca_prefill", "lca_mbp_step", "lca_generate", "lca_destroy"):
        assert n in names


def test_library_exports_every_declared_symbol():
    from paper_2608_15454_gb300 import build
    path = build.build()
    lib = ctypes.CDLL(path)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_covers_the_header():
    from paper_2608_15454_gb300 import lca
    assert set(declared_functions()) <= set(lca.EXPORTS)


def test_workspace_size_and_argument_checks_need_no_gpu():
    from paper_2608_15454_gb300 import build, lca
    from synth import PAPER, TINY
    build.build()
    lib = lca.load_library()
    n = ctypes.c_size_t()
    cfg = lca.make_config(TINY, 1, 400, 3)
    assert lib.lca_workspace_bytes(ctypes.byref(cfg), ctypes.byref(n)) == 0 and n.value > 0
    small = n.value
    cfg = lca.make_config(PAPER, 32, 2600, 4)
    assert lib.lca_workspace_bytes(ctypes.byref(cfg), ctypes.byref(n)) == 0 and n.value > small
    bad = lca.make_config(TINY, 1, 400, 3)
    bad.vocab = 300
    assert lib.lca_workspace_bytes(ctypes.byref(bad), ctypes.byref(n)) == -1
    bad = lca.make_config(TINY, 1, 400, 99)
    assert lib.lca_workspace_bytes(ctypes.byref(bad), ctypes.byref(n)) == -1
    assert lib.lca_mbp_step(None, 3, 0.5, 0, None, None) == -1
    assert lib.lca_status_str(-2) == b"capacity exceeded"
