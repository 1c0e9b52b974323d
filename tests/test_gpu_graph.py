"""The library's compute calls are graph-capturable (no allocation, no host
synchronization, every launch on the caller's stream): a whole denoise step
and commit, and a whole AR-Trust verify round, captured once into a CUDA graph
and replayed give the same bits as the same calls issued one by one."""
import math

import pytest
import torch

from gpu_helpers import gen, install_states, linear_desc, softmax_desc
from paper_2606_01774_gb300 import flare, workloads

pytestmark = pytest.mark.gpu
W = workloads.WORKLOADS


def _step_calls(w, outs, ws, st, verify=False, records=None):
    spec = w.spec
    ld = linear_desc(spec, w.state_pool.shape[0])
    b, sb = w.denoise[0], w.softmax[0]
    if verify:
        sd = softmax_desc(spec, w, flare.FLARE_MASK_ROW_TYPE_PER_REQUEST, w.row_type)
    else:
        sd = softmax_desc(spec, w)
    mv = spec.verify_horizon - 1

    def run():
        if verify:
            flare.check(flare.flare_verify_linear_attn(ld, mv, b.q, b.k, b.v, b.log_decay, b.beta,
                                                       w.state_pool, w.state_slot, w.verify_len,
                                                       outs[0], records, st))
        else:
            flare.check(flare.flare_block_linear_attn(ld, b.q, b.k, b.v, b.log_decay, b.beta,
                                                      w.state_pool, w.state_slot, outs[0], st))
        flare.check(flare.flare_block_softmax_attn(sd, sb.q, sb.k_blk, sb.v_blk, w.k_pool,
                                                   w.v_pool, w.page_table, w.prefix_len, outs[1],
                                                   outs[2], ws, ws.numel(), st))
        if verify:
            flare.check(flare.flare_verify_commit(ld, mv, [records], [w.state_pool], w.state_slot,
                                                  w.verify_accept, w.verify_len, st))
        else:
            c = w.commit
            flare.check(flare.flare_commit_state(ld, None, c.k, c.v, c.log_decay, c.beta,
                                                 w.state_pool, w.state_slot, w.accept_len, None,
                                                 st))
    return run, sd


@pytest.mark.parametrize("name", ["serving_batch64", "ar_trust_verify_batch64"])
def test_step_replays_bit_identically_from_a_graph(name):
    spec = W[name].replace(num_requests=8, prefix_lo=200, prefix_hi=2000)
    verify = spec.verify_horizon > 0
    w = gen(spec)
    install_states(w)
    pool0 = w.state_pool.clone()
    b, sb = w.denoise[0], w.softmax[0]
    outs = [torch.empty_like(b.v), torch.empty_like(sb.q),
            torch.empty(sb.q.shape[:3], dtype=torch.float32, device="cuda")]
    records = torch.zeros(spec.num_requests, max(spec.verify_horizon - 1, 1), spec.num_v_heads,
                          spec.head_dim_k, spec.head_dim_v, device="cuda") if verify else None
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    sd = softmax_desc(spec, w, flare.FLARE_MASK_ROW_TYPE_PER_REQUEST,
                      w.row_type) if verify else softmax_desc(spec, w)
    ws = torch.empty(max(flare.flare_softmax_workspace_size(sd), 256), dtype=torch.uint8,
                     device="cuda")
    run, _ = _step_calls(w, outs, ws, st, verify, records)

    # eager reference (the kernels' first launches also set their attributes)
    run()
    torch.cuda.synchronize()
    ref = [o.clone() for o in outs] + [w.state_pool.clone()]

    w.state_pool.copy_(pool0)
    for o in outs:
        o.zero_()
    side = torch.cuda.Stream()
    with torch.cuda.stream(side):
        g = torch.cuda.CUDAGraph()
        launches0 = flare.flare_launch_count()
        with torch.cuda.graph(g, stream=side):
            run()
        captured = flare.flare_launch_count() - launches0
    torch.cuda.synchronize()
    assert captured >= 4
    for _ in range(2):  # replay twice from the same starting pool
        w.state_pool.copy_(pool0)
        g.replay()
        torch.cuda.synchronize()
        for a, r in zip(outs + [w.state_pool], ref):
            assert torch.equal(a.view(torch.uint8), r.view(torch.uint8))
    assert flare.flare_read_status(st) == (flare.FLARE_OK, 0)
