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


def _gpc_model(ctas_per_sm, gpcs=8, sms_per_gpc=19):
    """Most clusters of c CTAs resident at once when a cluster must fit in one GPC."""
    return [0] + [gpcs * ((sms_per_gpc * ctas_per_sm) // c) for c in range(1, 17)]


def test_attention_grid_choice_on_the_host():
    """The cluster size the attention picks (host logic, no GPU) on a 152-SM, 8-GPC model:
    the sizes the measured 7B / 13B / batch-4 / 11-row workloads ran with."""
    import paper_2403_18647_gb300 as sd
    three, two = _gpc_model(3), _gpc_model(2)     # q <= 8: three CTAs per SM; q <= 16: two
    assert sd.attention_grid(32, three) == (11, 32)      # 7B, one sequence: 352 CTAs
    assert sd.attention_grid(40, three) == (9, 40)       # 13B: 360 CTAs
    assert sd.attention_grid(128, three) == (3, 128)     # 7B, four sequences: 384 CTAs
    assert sd.attention_grid(32, two) == (7, 32)         # 11-row blocks: 224 CTAs
    assert sd.attention_grid(512, three) == (1, 456)     # more pairs than fit: single CTAs
    assert sd.attention_grid(200, three) == (2, 200)
    assert sd.attention_grid(300, three) == (1, 300)
    assert sd.attention_grid(32, three, cs_cap=8) == (8, 32)
    assert sd.attention_grid(32, three, cs_cap=1) == (1, 32)
    assert sd.attention_grid(5, [0] * 17, num_sms=152) == (1, 5)     # no occupancy data: 2 per SM
    # a size the device cannot hold (0 clusters) is never chosen
    holes = list(three)
    holes[11] = holes[10] = 0
    assert sd.attention_grid(32, holes) == (9, 32)
    lib = sd.lib()
    assert lib.sdsat_attention_grid(0, None, 16, 152, None, None) == 1
