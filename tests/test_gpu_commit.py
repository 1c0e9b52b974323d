"""GPU parity of flare_commit_state against the oracle."""
import math

import numpy as np
import pytest
import torch

from gpu_helpers import (assert_out_close, assert_states_close, gen, install_states,
                         linear_desc, oracle_commit, reduced, run_commit, run_linear)
from paper_2606_01774_gb300 import flare, workloads

pytestmark = pytest.mark.gpu
W = workloads.WORKLOADS

CASES = {
    "tiny_fp32": W["tiny_fp32"],
    "single_request": W["single_request"],
    "small_model_batch256_r4": reduced(W["small_model_batch256"], 4),
    "multistep_batch128_r5": reduced(W["multistep_batch128"], 5, 100, 300),
    "ragged_block_b13": W["serving_batch64"].replace(num_requests=3, block_len=13, prefix_lo=0,
                                                     prefix_hi=70, accept="uniform", seed=31),
}


def ibits(t):
    return t.view(torch.int32)


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("causal", [False, True])
def test_commit_matches_oracle(name, causal):
    spec = CASES[name]
    w = gen(spec)
    install_states(w)
    before = w.state_pool.clone()
    pool = w.state_pool
    co = run_commit(w, pool, causal=causal)
    ref = oracle_commit(w, before, causal=causal)
    slots = w.state_slot.long()
    assert_states_close(pool[slots], ref["state"], name)
    if causal:
        assert_out_close(co, ref["causal"], spec.act_dtype, f"{name} causal")
    # slots that no request names stay bit-identical (they hold NaN)
    untouched = torch.ones(pool.shape[0], dtype=torch.bool, device=pool.device)
    untouched[slots] = False
    assert torch.equal(ibits(pool[untouched]), ibits(before[untouched]))
    # requests with accepted length 0 keep their state bit for bit
    zero = (w.accept_len == 0).nonzero().flatten()
    if len(zero):
        assert torch.equal(ibits(pool[slots[zero]]), ibits(before[slots[zero]]))


def test_accept_zero_is_bit_identical():
    spec = CASES["multistep_batch128_r5"]
    w = gen(spec)
    install_states(w)
    before = w.state_pool.clone()
    run_commit(w, w.state_pool, accept_len=torch.zeros_like(w.accept_len))
    assert torch.equal(ibits(w.state_pool), ibits(before))


def test_commit_full_block_agrees_with_denoise_readout():
    """Eq. noisy-block-fwd read from the commit side: the denoise output for a
    block equals s S_B^T q where S_B is the state the commit writes at r = B."""
    spec = CASES["small_model_batch256_r4"]
    w = gen(spec)
    install_states(w)
    w.denoise[0] = w.commit  # same block inputs for both calls
    out = run_linear(w, 0).double()
    pool = w.state_pool.clone()
    run_commit(w, pool, accept_len=torch.full_like(w.accept_len, spec.block_len))
    SB = pool[w.state_slot.long()].double()  # [R,Hv,dk,dv]
    q = w.commit.q.double()  # [R,B,Hk,dk]
    G = spec.num_v_heads // spec.num_qk_heads
    qv = q.repeat_interleave(G, dim=2)  # [R,B,Hv,dk]
    want = torch.einsum("rbhi,rhic->rbhc", qv, SB) / math.sqrt(spec.head_dim_k)
    err = (out - want).abs().max().item()
    assert err < 2e-2 and torch.linalg.norm(out - want) / torch.linalg.norm(want) < 1e-2


def test_commit_full_size_sampled():
    """multistep_batch128: 128 requests, accept lengths ~U[1,64], full launch."""
    spec = W["multistep_batch128"]
    w = gen(spec)
    R = spec.num_requests
    acc = w.accept_len.cpu()
    sample = sorted({0, R - 1, int(acc.argmin()), int(acc.argmax())})
    install_states(w, sample)
    before = w.state_pool.clone()
    run_commit(w, w.state_pool)
    ref = oracle_commit(w, before, sample)
    got = w.state_pool[w.state_slot.long()[sample]]
    assert_states_close(got, ref["state"], "multistep_batch128")
    assert torch.isfinite(w.state_pool[w.state_slot.long()]).all()


@pytest.mark.parametrize("name", ["serving_batch64", "small_model_batch256"])
def test_commit_full_size_every_request(name):
    """Full batch, every request's committed slot against the oracle; the slots
    no request uses keep their bits."""
    spec = W[name]
    w = gen(spec)
    install_states(w)
    before = w.state_pool.clone()
    run_commit(w, w.state_pool)
    ref = oracle_commit(w, before)
    got = w.state_pool[w.state_slot.long()]
    assert_states_close(got, ref["state"], name)
    used = torch.zeros(w.state_pool.shape[0], dtype=torch.bool, device=w.state_pool.device)
    used[w.state_slot.long()] = True
    assert torch.equal(w.state_pool[~used].view(torch.int32), before[~used].view(torch.int32))


@pytest.mark.parametrize("causal", [False, True])
def test_commit_strong_decay_folds_the_schedule(causal):
    """Log-gates of -3 per token drive the running decay below 2^-40 inside the
    block (the kernel then folds the decay into the state); half the heads keep
    the ordinary gates.  Same oracle, same tolerances."""
    spec = W["serving_batch64"].replace(num_requests=3, prefix_lo=0, prefix_hi=70,
                                        accept="uniform", seed=33)
    w = gen(spec)
    w.commit.log_decay[:, :, ::2] = -3.0
    install_states(w)
    before = w.state_pool.clone()
    co = run_commit(w, w.state_pool, causal=causal)
    ref = oracle_commit(w, before, causal=causal)
    slots = w.state_slot.long()
    assert_states_close(w.state_pool[slots], ref["state"], "strong decay")
    if causal:
        assert_out_close(co, ref["causal"], spec.act_dtype, "strong decay causal")
