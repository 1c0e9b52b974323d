"""Device-detected errors set status bits and skip the offending item; nothing
traps.  Invalid inputs here are ones the kernels' own range checks turn into a
status bit before any access (checked in the kernels' source)."""
import ctypes

import pytest
import torch

from gpu_helpers import gen, install_states, linear_desc, reduced, softmax_desc
from paper_2606_01774_gb300 import flare, workloads

pytestmark = pytest.mark.gpu
W = workloads.WORKLOADS


def _st():
    return torch.zeros(1, dtype=torch.int32, device="cuda")


def test_bounded_wait_gives_up_and_reports():
    """A pipeline wait on a barrier that nothing ever completes gives up after
    its limit (the same bounded wait every pipelined kernel uses) and reports
    FLARE_DEV_WAIT_TIMEOUT; the context stays usable."""
    import time

    st = _st()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    flare.check(flare.flare_debug_wait_timeout(st, 20_000_000), "flare_debug_wait_timeout")
    rc, bits = flare.flare_read_status(st)
    elapsed = time.perf_counter() - t0
    assert rc == flare.FLARE_ERR_DEVICE_STATUS and bits == flare.FLARE_DEV_WAIT_TIMEOUT
    assert elapsed >= 0.02
    # the context is intact: an ordinary call afterwards runs clean
    spec = reduced(W["serving_batch64"], 2, 64, 200)
    w = gen(spec)
    install_states(w)
    b = w.denoise[0]
    out = torch.empty_like(b.v)
    st2 = _st()
    flare.check(flare.flare_block_linear_attn(linear_desc(spec, w.state_pool.shape[0]), b.q, b.k,
                                              b.v, b.log_decay, b.beta, w.state_pool,
                                              w.state_slot, out, st2), "flare_block_linear_attn")
    assert flare.flare_read_status(st2) == (flare.FLARE_OK, 0)
    assert torch.isfinite(out.float()).all()


@pytest.mark.parametrize("name,args", [("small_model_batch256", ()),
                                       ("serving_batch64", (64, 200)),
                                       ("multistep_batch128", (100, 900))])
def test_bad_state_slot_sets_bit_and_skips_request(name, args):
    """Each denoise kernel (B = 16 and 32 persistent, B = 64 as one chunk)
    skips a request whose slot is out of range and flags it."""
    spec = reduced(W[name], 3, *args)
    w = gen(spec)
    install_states(w)
    nslots = w.state_pool.shape[0]
    w.state_slot[1] = nslots + 5
    blk = w.denoise[0]
    out = torch.full_like(blk.v, 7.0)
    st = _st()
    flare.check(flare.flare_block_linear_attn(linear_desc(spec, nslots), blk.q, blk.k, blk.v,
                                              blk.log_decay, blk.beta, w.state_pool,
                                              w.state_slot, out, st))
    rc, bits = flare.flare_read_status(st)
    assert rc == flare.FLARE_ERR_DEVICE_STATUS and bits == flare.FLARE_DEV_BAD_SLOT
    assert (out[1] == 7.0).all()
    assert (out[0] != 7.0).any() and (out[2] != 7.0).any()


def test_bad_accept_len_sets_bit_and_leaves_slot():
    spec = reduced(W["multistep_batch128"], 3, 64, 128)
    w = gen(spec)
    install_states(w)
    before = w.state_pool.clone()
    acc = w.accept_len.clone()
    acc[2] = spec.block_len + 1
    blk = w.commit
    st = _st()
    flare.check(flare.flare_commit_state(linear_desc(spec, w.state_pool.shape[0]), None, blk.k,
                                         blk.v, blk.log_decay, blk.beta, w.state_pool,
                                         w.state_slot, acc, None, st))
    rc, bits = flare.flare_read_status(st)
    assert bits == flare.FLARE_DEV_BAD_ACCEPT_LEN
    s2 = w.state_slot[2].long()
    assert torch.equal(w.state_pool[s2].view(torch.int32), before[s2].view(torch.int32))


@pytest.mark.parametrize("what", ["page", "prefix"])
def test_bad_page_or_prefix_sets_bit_and_skips_request(what):
    spec = reduced(W["serving_batch64"], 3, 200, 400)
    w = gen(spec)
    if what == "page":
        w.page_table[1, 1] = w.k_pool.shape[0]
        bit = flare.FLARE_DEV_BAD_PAGE
    else:
        w.prefix_len[1] = w.page_table.shape[1] * spec.page_size + 1
        bit = flare.FLARE_DEV_BAD_PREFIX_LEN
    sb = w.softmax[0]
    desc = softmax_desc(spec, w)
    nb = flare.flare_softmax_workspace_size(desc)
    ws = torch.empty(max(nb, 1), dtype=torch.uint8, device="cuda")
    out = torch.full_like(sb.q, 5.0)
    st = _st()
    flare.check(flare.flare_block_softmax_attn(desc, sb.q, sb.k_blk, sb.v_blk, w.k_pool,
                                               w.v_pool, w.page_table, w.prefix_len, out, None,
                                               ws, nb, st))
    rc, bits = flare.flare_read_status(st)
    assert rc == flare.FLARE_ERR_DEVICE_STATUS and bits == bit
    assert (out[1] == 5.0).all()
    assert torch.isfinite(out[0].float()).all() and (out[0] != 5.0).any()


def test_host_detected_errors_launch_nothing():
    spec = reduced(W["serving_batch64"], 2, 64, 128)
    w = gen(spec)
    sb = w.softmax[0]
    desc = softmax_desc(spec, w)
    nb = flare.flare_softmax_workspace_size(desc)
    out = torch.full_like(sb.q, 5.0)
    st = _st()
    # null output
    assert flare.flare_block_softmax_attn(desc, sb.q, sb.k_blk, sb.v_blk, w.k_pool, w.v_pool,
                                          w.page_table, w.prefix_len, None, None, None, nb,
                                          st) == flare.FLARE_ERR_INVALID_ARGUMENT
    # unsupported head dim
    bad = softmax_desc(spec, w)
    bad.head_dim = 96
    assert flare.flare_block_softmax_attn(bad, sb.q, sb.k_blk, sb.v_blk, w.k_pool, w.v_pool,
                                          w.page_table, w.prefix_len, out, None, None, 0,
                                          st) == flare.FLARE_ERR_UNSUPPORTED
    # block longer than 64
    bad = softmax_desc(spec, w)
    bad.block_len = 65
    assert flare.load().flare_block_softmax_attn(
        ctypes.byref(bad), None, None, None, None, None, None, None, None, None, None, 0,
        None, None) == flare.FLARE_ERR_UNSUPPORTED
    # workspace too small (only when the plan needs one)
    if nb:
        assert flare.flare_block_softmax_attn(desc, sb.q, sb.k_blk, sb.v_blk, w.k_pool,
                                              w.v_pool, w.page_table, w.prefix_len, out, None,
                                              None, nb - 1, st) == flare.FLARE_ERR_INVALID_ARGUMENT
    torch.cuda.synchronize()
    assert (out == 5.0).all()
    assert flare.flare_read_status(st) == (flare.FLARE_OK, 0)
