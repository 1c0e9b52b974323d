"""CPU checks of the C-ABI library: it builds, loads, exports every entry point
include/flare.h declares, and rejects bad arguments on the host before any
CUDA work (no compute call is made here)."""
import ctypes

import pytest

from paper_2606_01774_gb300 import build, flare


@pytest.fixture(scope="module")
def lib():
    build.build()
    return flare.load()


def test_header_declares_the_boundary():
    names = flare.declared_functions()
    for n in ("flare_block_linear_attn", "flare_commit_state", "flare_block_softmax_attn",
              "flare_softmax_workspace_size", "flare_debug_gather_prefix", "flare_read_status",
              "flare_status_string"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for n in flare.declared_functions():
        assert hasattr(lib, n), n


def test_status_strings(lib):
    assert flare.flare_status_string(0) == "FLARE_OK"
    assert flare.flare_status_string(4) == "FLARE_ERR_DEVICE_STATUS"


def test_host_argument_checks_need_no_gpu(lib):
    d = flare.linear_desc(2, 32, 16, 32, 128, 128, 6, flare.FLARE_DT_BF16, 0.088)
    null = [None] * 10
    assert lib.flare_block_linear_attn(ctypes.byref(d), *null) == flare.FLARE_ERR_INVALID_ARGUMENT
    d.head_dim_k = 96
    assert lib.flare_block_linear_attn(ctypes.byref(d), *null) == flare.FLARE_ERR_UNSUPPORTED
    d.head_dim_k = 128
    d.num_v_heads = 24
    d.num_qk_heads = 16
    assert lib.flare_block_linear_attn(ctypes.byref(d), *null) == flare.FLARE_ERR_INVALID_ARGUMENT
    assert lib.flare_block_linear_attn(None, *null) == flare.FLARE_ERR_INVALID_ARGUMENT
    s = flare.softmax_desc(2, 32, 16, 2, 256, 64, 100, 64, flare.FLARE_DT_BF16, 0.0625)
    s.mask_mode = 7
    n = ctypes.c_size_t(0)
    assert lib.flare_softmax_workspace_size(ctypes.byref(s), ctypes.byref(n)) == \
        flare.FLARE_ERR_INVALID_ARGUMENT
    s.mask_mode = 0
    s.page_size = 48
    assert lib.flare_softmax_workspace_size(ctypes.byref(s), ctypes.byref(n)) == \
        flare.FLARE_ERR_UNSUPPORTED
    assert lib.flare_read_status(None, None, None) == flare.FLARE_ERR_INVALID_ARGUMENT
    # the bounded-wait test entry rejects a missing status word and limits
    # outside 1 us .. 1 s before launching anything
    word = ctypes.c_int32(0)
    assert lib.flare_debug_wait_timeout(None, 1_000_000, None) == flare.FLARE_ERR_INVALID_ARGUMENT
    assert lib.flare_debug_wait_timeout(ctypes.byref(word), 999, None) == \
        flare.FLARE_ERR_INVALID_ARGUMENT
    assert lib.flare_debug_wait_timeout(ctypes.byref(word), 2_000_000_000, None) == \
        flare.FLARE_ERR_INVALID_ARGUMENT


def test_workspace_query_is_host_only(lib):
    s = flare.softmax_desc(1, 32, 16, 2, 256, 64, 100, 64, flare.FLARE_DT_BF16, 0.0625)
    n = flare.flare_softmax_workspace_size(s)
    assert n >= 0 and n % 256 == 0
    s.num_requests = 0
    assert flare.flare_softmax_workspace_size(s) == 0


def _header_param_counts():
    """Parameter count of every entry point declared in include/flare.h."""
    import re

    text = re.sub(r"/\*.*?\*/", "", flare.HEADER.read_text(), flags=re.S)
    counts = {}
    for m in re.finditer(r"\b(flare_\w+)\s*\(([^;{]*?)\)\s*;", text, re.S):
        args = m.group(2).strip()
        counts[m.group(1)] = 0 if args in ("", "void") else args.count(",") + 1
    return counts


def test_binding_signatures_match_the_header(lib):
    """The ctypes argument lists of the binding have as many entries as the
    declarations in the header have parameters."""
    counts = _header_param_counts()
    assert "flare_verify_linear_attn" in counts and "flare_verify_commit" in counts
    for name, n in counts.items():
        fn = getattr(lib, name)
        if fn.argtypes is not None:
            assert len(fn.argtypes) == n, (name, len(fn.argtypes), n)


def test_verify_entry_points_check_arguments_on_the_host(lib):
    d = flare.linear_desc(2, 31, 16, 32, 128, 128, 6, flare.FLARE_DT_BF16, 0.088)
    assert lib.flare_verify_linear_attn(ctypes.byref(d), 15, *([None] * 12)) == \
        flare.FLARE_ERR_INVALID_ARGUMENT
    assert lib.flare_verify_linear_attn(ctypes.byref(d), -1, *([None] * 12)) == \
        flare.FLARE_ERR_INVALID_ARGUMENT
    assert lib.flare_verify_commit(ctypes.byref(d), 15, 0, *([None] * 7)) == \
        flare.FLARE_ERR_INVALID_ARGUMENT
    assert lib.flare_verify_commit(ctypes.byref(d), 15, 65, *([None] * 7)) == \
        flare.FLARE_ERR_UNSUPPORTED
    s = flare.softmax_desc(2, 31, 16, 2, 256, 64, 100, 64, flare.FLARE_DT_BF16, 0.0625,
                           flare.FLARE_MASK_ROW_TYPE_PER_REQUEST, None)
    n = ctypes.c_size_t(0)
    assert lib.flare_softmax_workspace_size(ctypes.byref(s), ctypes.byref(n)) == \
        flare.FLARE_ERR_INVALID_ARGUMENT
    s.mask_mode = 4
    assert lib.flare_softmax_workspace_size(ctypes.byref(s), ctypes.byref(n)) == \
        flare.FLARE_ERR_INVALID_ARGUMENT
