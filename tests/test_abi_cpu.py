"""The C ABI library builds, loads without a GPU and exports every declared entry point."""
import ctypes
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "sdsat.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(sdsat_[a-z_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("sdsat_create", "sdsat_destroy", "sdsat_kv_create", "sdsat_block_forward",
              "sdsat_accept_greedy", "sdsat_accept_nucleus", "sdsat_kv_commit", "sdsat_status_string",
              "sdsat_block_forward_tree", "sdsat_accept_tree", "sdsat_build_tree_block",
              "sdsat_build_pipelined_block", "sdsat_accept_pipelined"):
        assert n in names


def test_library_exports_every_declared_symbol():
    from paper_2403_18647_gb300 import build as b
    if b.is_stale():
        b.build()
    lib = ctypes.CDLL(b.LIB)
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert not missing, missing


def test_status_strings_without_gpu():
    import paper_2403_18647_gb300 as sd
    lib = sd.lib()
    assert lib.sdsat_status_string(0) == b"ok"
    assert lib.sdsat_status_string(1) == b"invalid argument"


def test_argument_errors_are_synchronous_and_need_no_gpu():
    """Null handles are rejected on the host before any CUDA call."""
    import paper_2403_18647_gb300 as sd
    lib = sd.lib()
    assert lib.sdsat_block_forward(None, None, None, None, 1, 6, None) == 1
    assert lib.sdsat_accept_greedy(None, None, None, None, 1, 6, 0, None, None, 1) == 1
    assert lib.sdsat_create(None, None, None, None) == 1
    assert lib.sdsat_block_forward_tree(None, None, None, None, 1, 7, None) == 1
    assert lib.sdsat_accept_tree(None, None, None, None, None, 1, 7, 0.0, 1.0, 0, 0, None, None, None, 1) == 1
    assert lib.sdsat_build_tree_block(None, None, 2, None, 4, None, None, 2, 0, 1, 3, None) == 1
    assert lib.sdsat_build_pipelined_block(None, None, None, None, None, None, None, 0, 1, 5, None) == 1
    assert lib.sdsat_accept_pipelined(None, None, None, None, None, 1, 11, 0.0, 1.0, 0, 0, None, None, 1) == 1
