"""The library's compute calls are graph-capturable (no allocation, no host
synchronization, every launch on the caller's stream): a whole denoise step
and commit, a whole AR-Trust verify round, the two-stream training forward and
a ShortConv denoise + commit, captured once into a CUDA graph and replayed,
give the same bits as the same calls issued one by one."""
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


def _replays_like_eager(run, outs, states=()):
    """Issues `run` once eagerly, then captures it into a CUDA graph and
    replays it twice from the same starting states: the outputs and states
    must come back bit for bit."""
    starts = [s.clone() for s in states]
    run()
    torch.cuda.synchronize()
    ref = [t.clone() for t in list(outs) + list(states)]
    for s, s0 in zip(states, starts):
        s.copy_(s0)
    side = torch.cuda.Stream()
    with torch.cuda.stream(side):
        g = torch.cuda.CUDAGraph()
        launches0 = flare.flare_launch_count()
        with torch.cuda.graph(g, stream=side):
            run()
        captured = flare.flare_launch_count() - launches0
    torch.cuda.synchronize()
    assert captured >= 1
    for _ in range(2):
        for s, s0 in zip(states, starts):
            s.copy_(s0)
        for o in outs:
            o.zero_()
        g.replay()
        torch.cuda.synchronize()
        for a, r in zip(list(outs) + list(states), ref):
            assert torch.equal(a.view(torch.uint8), r.view(torch.uint8))


def test_two_stream_replays_bit_identically_from_a_graph():
    sp = workloads.TWO_STREAM_WORKLOADS["two_stream_train_b4"].replace(
        num_seqs=1, seq_len=256, num_qk_heads=2, num_v_heads=4, seed=31)
    x = workloads.generate_two_stream(sp, "cuda")
    gen_ = torch.Generator(device="cuda")
    gen_.manual_seed(5)
    cs = 0.05 * torch.randn(sp.num_seqs, sp.num_v_heads, sp.seq_len // sp.chunk_len, 128, 128,
                            generator=gen_, device="cuda")
    d = flare.two_stream_desc(sp.num_seqs, sp.seq_len, sp.chunk_len, sp.block_len,
                              sp.num_qk_heads, sp.num_v_heads, 128, 128, flare.FLARE_DT_BF16,
                              1.0 / math.sqrt(128))
    out = torch.empty_like(x.noisy.v)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    c, nz = x.clean, x.noisy

    def run():
        flare.check(flare.flare_two_stream_fwd(d, cs, c.k, c.v, c.log_decay, c.beta, nz.q, nz.k,
                                               nz.v, nz.log_decay, nz.beta, out, st))

    _replays_like_eager(run, [out])
    assert flare.flare_read_status(st) == (flare.FLARE_OK, 0)


def test_shortconv_denoise_and_commit_replay_bit_identically_from_a_graph():
    spec = W["shortconv_serving_batch64"].replace(num_requests=6, prefix_lo=64, prefix_hi=128)
    w = gen(spec)
    act = flare.FLARE_DT_BF16
    d = flare.conv_desc(spec.num_requests, spec.block_len, spec.conv_channels, spec.conv_width,
                        w.conv_state.shape[0], act, flare.FLARE_ACT_SILU)
    x0, x1 = w.conv_x[0], w.conv_commit_x
    out0, out1 = torch.empty_like(x0), torch.empty_like(x1)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")

    def run():
        flare.check(flare.flare_short_conv(d, x0, w.conv_state, w.state_slot, w.conv_weight,
                                           w.conv_bias, None, out0, st))
        flare.check(flare.flare_short_conv(d, x1, w.conv_state, w.state_slot, w.conv_weight,
                                           w.conv_bias, w.accept_len, out1, st))

    _replays_like_eager(run, [out0, out1], [w.conv_state])
    assert flare.flare_read_status(st) == (flare.FLARE_OK, 0)
