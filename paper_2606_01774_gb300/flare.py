"""Thin ctypes binding of ``libflare.so`` (declared in ``include/flare.h``).

Argument marshalling only: every function takes torch tensors that already
live on the current CUDA device (or None for nullable arguments), passes their
data pointers and the stream to the C entry point of the same name, and
returns the ``flare_status`` code.  No arithmetic of the method happens here,
and there is no fallback: if the library is missing or was built for another
machine, loading it raises.
"""
from __future__ import annotations

import ctypes
import re
from pathlib import Path

_PKG = Path(__file__).resolve().parent
LIB_PATH = _PKG / "libflare.so"
HEADER = _PKG.parent / "include" / "flare.h"

FLARE_OK = 0
FLARE_ERR_INVALID_ARGUMENT = 1
FLARE_ERR_UNSUPPORTED = 2
FLARE_ERR_CUDA = 3
FLARE_ERR_DEVICE_STATUS = 4

FLARE_DT_BF16 = 0
FLARE_DT_F32 = 1
FLARE_MASK_BLOCK_BIDIR = 0
FLARE_MASK_BLOCK_CAUSAL = 1
FLARE_MASK_ROW_TYPE_UNIFORM = 2
FLARE_MASK_ROW_TYPE_PER_REQUEST = 3
FLARE_ROW_CAUSAL = 0
FLARE_ROW_BIDIR = 1
FLARE_ACT_NONE = 0
FLARE_ACT_SILU = 1

FLARE_DEV_BAD_SLOT = 0x1
FLARE_DEV_BAD_PAGE = 0x2
FLARE_DEV_BAD_PREFIX_LEN = 0x4
FLARE_DEV_BAD_ACCEPT_LEN = 0x8
FLARE_DEV_WAIT_TIMEOUT = 0x10
FLARE_DEV_BAD_VERIFY_LEN = 0x20


class FlareError(RuntimeError):
    def __init__(self, status, what=""):
        self.status = status
        super().__init__(f"{what}: {flare_status_string(status)}" if what else
                         flare_status_string(status))


class flare_linear_desc(ctypes.Structure):
    _fields_ = [("num_requests", ctypes.c_int32), ("block_len", ctypes.c_int32),
                ("num_qk_heads", ctypes.c_int32), ("num_v_heads", ctypes.c_int32),
                ("head_dim_k", ctypes.c_int32), ("head_dim_v", ctypes.c_int32),
                ("num_state_slots", ctypes.c_int32), ("act_dtype", ctypes.c_int),
                ("scale", ctypes.c_float)]


class flare_conv_desc(ctypes.Structure):
    _fields_ = [("num_requests", ctypes.c_int32), ("block_len", ctypes.c_int32),
                ("channels", ctypes.c_int32), ("width", ctypes.c_int32),
                ("num_state_slots", ctypes.c_int32), ("act_dtype", ctypes.c_int),
                ("activation", ctypes.c_int)]


class flare_two_stream_desc(ctypes.Structure):
    _fields_ = [("num_seqs", ctypes.c_int32), ("seq_len", ctypes.c_int32),
                ("chunk_len", ctypes.c_int32), ("block_len", ctypes.c_int32),
                ("num_qk_heads", ctypes.c_int32), ("num_v_heads", ctypes.c_int32),
                ("head_dim_k", ctypes.c_int32), ("head_dim_v", ctypes.c_int32),
                ("act_dtype", ctypes.c_int), ("scale", ctypes.c_float)]


class flare_softmax_desc(ctypes.Structure):
    _fields_ = [("num_requests", ctypes.c_int32), ("block_len", ctypes.c_int32),
                ("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("num_pages", ctypes.c_int32), ("max_pages_per_req", ctypes.c_int32),
                ("act_dtype", ctypes.c_int), ("scale", ctypes.c_float),
                ("mask_mode", ctypes.c_int), ("row_type", ctypes.c_void_p)]


_lib = None


def load() -> ctypes.CDLL:
    """Load libflare.so (raises OSError if it is missing: there is no fallback)."""
    global _lib
    if _lib is not None:
        return _lib
    if not LIB_PATH.exists():
        raise OSError(f"{LIB_PATH} is missing; build it with paper_2606_01774_gb300.build.build()")
    lib = ctypes.CDLL(str(LIB_PATH))
    P, S, I32 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int32
    lin = ctypes.POINTER(flare_linear_desc)
    smx = ctypes.POINTER(flare_softmax_desc)
    cnv = ctypes.POINTER(flare_conv_desc)
    tsd = ctypes.POINTER(flare_two_stream_desc)
    sigs = {
        "flare_short_conv": [cnv] + [P] * 9,
        "flare_two_stream_fwd": [tsd] + [P] * 13,
        "flare_block_linear_attn": [lin] + [P] * 10,
        "flare_commit_state": [lin] + [P] * 11,
        "flare_verify_linear_attn": [lin, I32] + [P] * 12,
        "flare_verify_commit": [lin, I32, I32] + [P] * 7,
        "flare_softmax_workspace_size": [smx, ctypes.POINTER(S)],
        "flare_block_softmax_attn": [smx] + [P] * 10 + [S, P, P],
        "flare_block_softmax_attn_noalloc": [smx] + [P] * 11,
        "flare_append_kv": [smx] + [P] * 9,
        "flare_debug_gather_prefix": [smx, P, P, P, P, I32, P, P, P, P],
        "flare_debug_wait_timeout": [P, ctypes.c_uint64, P],
        "flare_read_status": [P, P, ctypes.POINTER(I32)],
    }
    for name, args in sigs.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = ctypes.c_int
    lib.flare_launch_count.argtypes = []
    lib.flare_launch_count.restype = ctypes.c_uint64
    lib.flare_status_string.argtypes = [ctypes.c_int]
    lib.flare_status_string.restype = ctypes.c_char_p
    _lib = lib
    return lib


def declared_functions():
    """Names of the entry points declared in include/flare.h."""
    text = HEADER.read_text()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w\s\*]*?\b(flare_\w+)\s*\(", text, re.M)))


def _p(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch

        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(getattr(stream, "cuda_stream", stream))


def flare_launch_count() -> int:
    return int(load().flare_launch_count())


def flare_status_string(status: int) -> str:
    return load().flare_status_string(int(status)).decode()


def check(status: int, what: str = "") -> None:
    if status != FLARE_OK:
        raise FlareError(status, what)


def flare_block_linear_attn(desc, q, k, v, log_decay, beta, state_pool, state_slot, out,
                            dev_status, stream=None) -> int:
    return load().flare_block_linear_attn(
        ctypes.byref(desc), _p(q), _p(k), _p(v), _p(log_decay), _p(beta), _p(state_pool),
        _p(state_slot), _p(out), _p(dev_status), _stream(stream))


def flare_commit_state(desc, q, k, v, log_decay, beta, state_pool, state_slot, accept_len,
                       causal_out, dev_status, stream=None) -> int:
    return load().flare_commit_state(
        ctypes.byref(desc), _p(q), _p(k), _p(v), _p(log_decay), _p(beta), _p(state_pool),
        _p(state_slot), _p(accept_len), _p(causal_out), _p(dev_status), _stream(stream))


def flare_verify_linear_attn(desc, max_verify, q, k, v, log_decay, beta, state_pool,
                             state_slot, verify_len, out, verify_states, dev_status,
                             stream=None) -> int:
    return load().flare_verify_linear_attn(
        ctypes.byref(desc), int(max_verify), _p(q), _p(k), _p(v), _p(log_decay), _p(beta),
        _p(state_pool), _p(state_slot), _p(verify_len), _p(out), _p(verify_states),
        _p(dev_status), _stream(stream))


def flare_verify_commit(desc, max_verify, verify_states, state_pools, state_slot, accept,
                        verify_len, dev_status, stream=None) -> int:
    """verify_states, state_pools: sequences of per-layer device tensors; their
    data pointers are passed as host arrays."""
    n = len(state_pools)
    recs = (ctypes.c_void_p * n)(*[None if t is None else t.data_ptr() for t in verify_states])
    pools = (ctypes.c_void_p * n)(*[t.data_ptr() for t in state_pools])
    return load().flare_verify_commit(
        ctypes.byref(desc), int(max_verify), n, recs, pools, _p(state_slot), _p(accept),
        _p(verify_len), _p(dev_status), _stream(stream))


def flare_short_conv(desc, x, conv_state, state_slot, weight, bias, accept_len, out,
                     dev_status, stream=None) -> int:
    return load().flare_short_conv(
        ctypes.byref(desc), _p(x), _p(conv_state), _p(state_slot), _p(weight), _p(bias),
        _p(accept_len), _p(out), _p(dev_status), _stream(stream))


def flare_two_stream_fwd(desc, chunk_states, k, v, log_decay, beta, q_noisy, k_noisy, v_noisy,
                         log_decay_noisy, beta_noisy, out_noisy, dev_status, stream=None) -> int:
    return load().flare_two_stream_fwd(
        ctypes.byref(desc), _p(chunk_states), _p(k), _p(v), _p(log_decay), _p(beta), _p(q_noisy),
        _p(k_noisy), _p(v_noisy), _p(log_decay_noisy), _p(beta_noisy), _p(out_noisy),
        _p(dev_status), _stream(stream))


def flare_softmax_workspace_size(desc) -> int:
    n = ctypes.c_size_t(0)
    check(load().flare_softmax_workspace_size(ctypes.byref(desc), ctypes.byref(n)),
          "flare_softmax_workspace_size")
    return int(n.value)


def flare_block_softmax_attn(desc, q, k_blk, v_blk, k_pool, v_pool, page_table, prefix_len,
                             out, lse, workspace, workspace_bytes, dev_status, stream=None) -> int:
    return load().flare_block_softmax_attn(
        ctypes.byref(desc), _p(q), _p(k_blk), _p(v_blk), _p(k_pool), _p(v_pool), _p(page_table),
        _p(prefix_len), _p(out), _p(lse), _p(workspace), int(workspace_bytes), _p(dev_status),
        _stream(stream))


def flare_append_kv(desc, k_blk, v_blk, k_pool, v_pool, page_table, prefix_len, append_len,
                    dev_status, stream=None) -> int:
    return load().flare_append_kv(
        ctypes.byref(desc), _p(k_blk), _p(v_blk), _p(k_pool), _p(v_pool), _p(page_table),
        _p(prefix_len), _p(append_len), _p(dev_status), _stream(stream))


FLARE_NOALLOC_SCRATCH_BYTES = 64 * 1024 * 1024


def flare_block_softmax_attn_noalloc(desc, q, k_blk, v_blk, k_pool, v_pool, page_table,
                                     prefix_len, out, lse, dev_status, stream=None) -> int:
    return load().flare_block_softmax_attn_noalloc(
        ctypes.byref(desc), _p(q), _p(k_blk), _p(v_blk), _p(k_pool), _p(v_pool), _p(page_table),
        _p(prefix_len), _p(out), _p(lse), _p(dev_status), _stream(stream))


def flare_debug_gather_prefix(desc, k_pool, v_pool, page_table, prefix_len, request, k_out,
                              v_out, dev_status, stream=None) -> int:
    return load().flare_debug_gather_prefix(
        ctypes.byref(desc), _p(k_pool), _p(v_pool), _p(page_table), _p(prefix_len),
        int(request), _p(k_out), _p(v_out), _p(dev_status), _stream(stream))


def flare_debug_wait_timeout(dev_status, limit_ns, stream=None) -> int:
    return load().flare_debug_wait_timeout(_p(dev_status), int(limit_ns), _stream(stream))


def flare_read_status(dev_status, stream=None):
    """Returns (status, bits)."""
    bits = ctypes.c_int32(0)
    st = load().flare_read_status(_p(dev_status), _stream(stream), ctypes.byref(bits))
    return st, int(bits.value)


# ---------------------------------------------------------------- descriptors


def linear_desc(num_requests, block_len, num_qk_heads, num_v_heads, head_dim_k, head_dim_v,
                num_state_slots, act_dtype, scale) -> flare_linear_desc:
    return flare_linear_desc(num_requests, block_len, num_qk_heads, num_v_heads, head_dim_k,
                             head_dim_v, num_state_slots, act_dtype, scale)


def conv_desc(num_requests, block_len, channels, width, num_state_slots, act_dtype,
              activation=FLARE_ACT_SILU) -> flare_conv_desc:
    return flare_conv_desc(num_requests, block_len, channels, width, num_state_slots, act_dtype,
                           activation)


def two_stream_desc(num_seqs, seq_len, chunk_len, block_len, num_qk_heads, num_v_heads,
                    head_dim_k, head_dim_v, act_dtype, scale) -> flare_two_stream_desc:
    return flare_two_stream_desc(num_seqs, seq_len, chunk_len, block_len, num_qk_heads,
                                 num_v_heads, head_dim_k, head_dim_v, act_dtype, scale)


def softmax_desc(num_requests, block_len, num_q_heads, num_kv_heads, head_dim, page_size,
                 num_pages, max_pages_per_req, act_dtype, scale,
                 mask_mode=FLARE_MASK_BLOCK_BIDIR, row_type=None) -> flare_softmax_desc:
    """row_type: uint8 device tensor ([B] or [R,B]) for the ROW_TYPE mask modes;
    the caller keeps it alive while the descriptor is in use."""
    return flare_softmax_desc(num_requests, block_len, num_q_heads, num_kv_heads, head_dim,
                              page_size, num_pages, max_pages_per_req, act_dtype, scale, mask_mode,
                              None if row_type is None else row_type.data_ptr())
