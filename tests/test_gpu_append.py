"""GPU KV append (state-update pass) against the oracle: bit-exact page writes."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import gen, softmax_desc
from paper_2606_01774_gb300 import flare, workloads

pytestmark = pytest.mark.gpu
W = workloads.WORKLOADS


def _with_room(spec):
    """Workload whose page tables name pages for the block after each prefix."""
    w = gen(spec)
    R, B, p = spec.num_requests, spec.block_len, spec.page_size
    table = w.page_table.cpu().numpy()
    lens = w.prefix_len.cpu().numpy()
    need = [max(0, -(-(int(P) + B) // p) - (-(-int(P) // p))) for P in lens]
    extra = sum(need)
    num_pages = w.k_pool.shape[0]
    pad = torch.full((extra,) + tuple(w.k_pool.shape[1:]), float("nan"), dtype=w.k_pool.dtype,
                     device="cuda")
    w.k_pool = torch.cat([w.k_pool, pad]).contiguous()
    w.v_pool = torch.cat([w.v_pool, pad.clone()]).contiguous()
    cols = max(table.shape[1], max(-(-(int(P) + B) // p) for P in lens))
    t2 = -np.ones((R, cols), np.int32)
    t2[:, :table.shape[1]] = table
    nxt = num_pages
    for r, P in enumerate(lens):
        for q in range(-(-int(P) // p), -(-(int(P) + B) // p)):
            t2[r, q] = nxt
            nxt += 1
    w.page_table = torch.from_numpy(t2).cuda().contiguous()
    return w


def _bits(t):
    return t.view(torch.int16) if t.element_size() == 2 else t.view(torch.int32)


@pytest.mark.parametrize("name", ["tiny_fp32", "serving_batch64", "small_model_batch256"])
@pytest.mark.parametrize("partial", [False, True])
def test_append_matches_oracle_bit_for_bit(name, partial):
    spec = W[name].replace(num_requests=min(W[name].num_requests, 6), prefix_lo=1,
                           prefix_hi=min(W[name].prefix_hi, 700), seed=55)
    w = _with_room(spec)
    sb = w.softmax[0]
    acc = None
    if partial:
        g = torch.Generator(device="cuda")
        g.manual_seed(3)
        acc = torch.randint(0, spec.block_len + 1, (spec.num_requests,), generator=g,
                            device="cuda", dtype=torch.int32)
    kp_ref, vp_ref = oracle.append_kv(sb.k_blk.cpu(), sb.v_blk.cpu(), w.k_pool.cpu(),
                                      w.v_pool.cpu(), w.page_table.cpu(), w.prefix_len.cpu(),
                                      None if acc is None else acc.cpu())
    desc = softmax_desc(spec, w)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    flare.check(flare.flare_append_kv(desc, sb.k_blk, sb.v_blk, w.k_pool, w.v_pool, w.page_table,
                                      w.prefix_len, acc, st))
    assert flare.flare_read_status(st) == (flare.FLARE_OK, 0)
    for got, ref in ((w.k_pool, kp_ref), (w.v_pool, vp_ref)):
        g = _bits(got).cpu().numpy()
        assert np.array_equal(g.view(np.uint8), np.ascontiguousarray(ref).view(np.uint8))


def test_append_then_softmax_sees_the_block_in_the_prefix():
    """After appending a block and advancing prefix_len, a softmax over the
    longer prefix with a 1-token block equals the oracle on the same inputs."""
    spec = W["serving_batch64"].replace(num_requests=3, prefix_lo=100, prefix_hi=300, seed=56)
    w = _with_room(spec)
    sb = w.softmax[0]
    desc = softmax_desc(spec, w)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    flare.check(flare.flare_append_kv(desc, sb.k_blk, sb.v_blk, w.k_pool, w.v_pool, w.page_table,
                                      w.prefix_len, None, st))
    w.prefix_len += spec.block_len
    for r in range(spec.num_requests):
        got = oracle.gather_prefix(r, w.k_pool.cpu(), w.page_table.cpu(), w.prefix_len.cpu(),
                                   spec.page_size)
        tail = got[-spec.block_len:]
        assert np.array_equal(tail, sb.k_blk[r].double().cpu().numpy())


def test_append_range_errors_skip_the_request():
    spec = W["serving_batch64"].replace(num_requests=3, prefix_lo=100, prefix_hi=300, seed=57)
    w = _with_room(spec)
    before_k = w.k_pool.clone()
    acc = torch.full((3,), 4, dtype=torch.int32, device="cuda")
    acc[1] = spec.block_len + 1
    sb = w.softmax[0]
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    flare.check(flare.flare_append_kv(softmax_desc(spec, w), sb.k_blk, sb.v_blk, w.k_pool,
                                      w.v_pool, w.page_table, w.prefix_len, acc, st))
    rc, bits = flare.flare_read_status(st)
    assert bits == flare.FLARE_DEV_BAD_ACCEPT_LEN
    # request 1 untouched: its would-be rows still hold the old bits
    P = int(w.prefix_len[1])
    pg = int(w.page_table[1, P // spec.page_size])
    assert torch.equal(_bits(w.k_pool[pg]), _bits(before_k[pg]))
