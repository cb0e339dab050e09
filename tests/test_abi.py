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


def test_workspace_is_sized_by_cache_pages():
    """Every cache layer is a pool of 64-slot pages [pages][H][64][hd]: a page of one layer holds
    K and V of 64 positions, 64 x d x 2 values (256 KB at d = 1024 in bf16). Each encoder and
    next-byte layer's pool has kv_pages pages, each LM layer's lm_pages, each multi-byte layer's
    mb_pages; 0 sizes a pool for every sequence at max_bytes."""
    from paper_2608_15454_gb300 import build, lca
    from synth import PAPER
    build.build()
    lib = lca.load_library()
    n = ctypes.c_size_t()

    def ws(**kw):
        cfg = lca.make_config(PAPER, 8, 8192, 4, **kw)
        assert lib.lca_workspace_bytes(ctypes.byref(cfg), ctypes.byref(n)) == 0
        return n.value

    page = 64 * PAPER.d_model * 2 * 2
    full = ws()
    pages_byte = 8 * 8192 // 64        # 8 sequences x 128 pages
    pages_lm = 8 * ((8192 + 1 + 63) // 64)
    byte_layers = PAPER.n_enc + PAPER.n_nb
    assert full - ws(kv_pages=100) == (pages_byte - 100) * byte_layers * page
    assert full - ws(lm_pages=100) == (pages_lm - 100) * PAPER.n_lm * page
    assert full - ws(mb_pages=100) == (pages_byte - 100) * PAPER.n_mb * page
    # the explicit worst case is the default
    assert ws(kv_pages=pages_byte, lm_pages=pages_lm, mb_pages=pages_byte) == full
    # an LM cache of 16 pages per sequence (1,024 latents) instead of 129: 16 layers x 113 x 8 pages less
    assert full - ws(lm_pages=8 * 16) == 8 * 113 * PAPER.n_lm * page
    for bad in ({"kv_pages": -1}, {"lm_pages": -5}, {"mb_pages": -1}):
        cfg = lca.make_config(PAPER, 8, 8192, 4, **bad)
        assert lib.lca_workspace_bytes(ctypes.byref(cfg), ctypes.byref(n)) == -1
    # the page table row of a sequence is staged in shared memory: at most 2,048 pages
    cfg = lca.make_config(PAPER, 1, 131071, 4)
    assert lib.lca_workspace_bytes(ctypes.byref(cfg), ctypes.byref(n)) == 0
    cfg = lca.make_config(PAPER, 1, 131072, 4)
    assert lib.lca_workspace_bytes(ctypes.byref(cfg), ctypes.byref(n)) == -1
