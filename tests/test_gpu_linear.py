"""GPU parity of flare_block_linear_attn (denoise pass) against the oracle."""
import math

import numpy as np
import pytest
import torch

from gpu_helpers import (assert_out_close, gen, install_states, oracle_linear, reduced,
                         run_linear)
from paper_2606_01774_gb300 import flare, workloads

pytestmark = pytest.mark.gpu
W = workloads.WORKLOADS

CASES = {
    "tiny_fp32": W["tiny_fp32"],
    "single_request": W["single_request"],
    "serving_batch64_r3": reduced(W["serving_batch64"], 3, 512, 1500),
    "small_model_batch256_r4": reduced(W["small_model_batch256"], 4),
    "multistep_batch128_r3": reduced(W["multistep_batch128"], 3, 100, 900),
    "ragged_block_b13": W["serving_batch64"].replace(num_requests=2, block_len=13, prefix_lo=0,
                                                     prefix_hi=70, seed=21),
    "d64_bf16": W["tiny_fp32"].replace(act_dtype="bf16", num_requests=3, num_v_heads=4,
                                       block_len=40, seed=22),
    # 33..64 rows: the block as one chunk, rows past B zero
    "ragged_block_b45": W["serving_batch64"].replace(num_requests=3, block_len=45, prefix_lo=0,
                                                     prefix_hi=70, seed=23),
    "ragged_block_b33": W["serving_batch64"].replace(num_requests=2, block_len=33, prefix_lo=0,
                                                     prefix_hi=70, seed=24),
    # more (request, value head) items than the persistent kernel's CTAs, so
    # that CTAs walk a second item with a ragged block
    "ragged_block_b50_r12": W["serving_batch64"].replace(num_requests=12, block_len=50,
                                                         prefix_lo=0, prefix_hi=70, seed=25),
    "ragged_block_b27_r12": W["serving_batch64"].replace(num_requests=12, block_len=27,
                                                         prefix_lo=0, prefix_hi=70, seed=26),
}


def bits(t):
    return t.view(torch.int32) if t.dtype == torch.float32 else t.view(torch.int16)


@pytest.mark.parametrize("name", list(CASES))
def test_denoise_matches_oracle(name):
    spec = CASES[name]
    w = gen(spec)
    install_states(w)
    before = w.state_pool.clone()
    for step in range(min(2, spec.denoise_steps)):
        out = run_linear(w, step)
        ref = oracle_linear(w, step)
        assert_out_close(out, ref, spec.act_dtype, f"{name} step {step}")
    # the denoise pass reads the pool and never writes it (NaN slots included)
    assert torch.equal(bits(w.state_pool), bits(before))


@pytest.mark.parametrize("name", ["serving_batch64", "small_model_batch256", "multistep_batch128"])
def test_denoise_full_size_sampled(name):
    """Full batch, the launch configuration bench.py times; the oracle checks a
    sample of requests element by element."""
    spec = W[name]
    w = gen(spec)
    R = spec.num_requests
    sample = sorted({0, R // 2, R - 1})
    install_states(w, sample)
    out = run_linear(w, spec.denoise_steps - 1)
    assert torch.isfinite(out).all()
    ref = oracle_linear(w, spec.denoise_steps - 1, sample)
    assert_out_close(out[sample], ref, spec.act_dtype, name)


@pytest.mark.parametrize("name", ["serving_batch64", "small_model_batch256"])
def test_denoise_full_size_every_request(name):
    """Full batch in the launch configuration bench.py times, every request and
    head element by element against the per-token recurrence."""
    spec = W[name]
    w = gen(spec)
    install_states(w)
    out = run_linear(w, spec.denoise_steps - 1)
    ref = oracle_linear(w, spec.denoise_steps - 1)
    assert_out_close(out, ref, spec.act_dtype, name)


@pytest.mark.parametrize("name", ["serving_batch64_r3", "small_model_batch256_r4",
                                  "multistep_batch128_r3", "d64_bf16"])
def test_denoise_strong_decay(name):
    """Log-gates of -3 per token on every other value head: the block's running
    decay falls below the fp32 range inside the block (Gam_{B-1} is 0 in fp32 at
    B = 64) and the masked exponentials of A and M2 overflow; half the heads
    keep the ordinary gates.  Same oracle, same tolerances."""
    spec = CASES[name]
    w = gen(spec)
    w.denoise[0].log_decay[:, :, ::2] = -3.0
    install_states(w)
    out = run_linear(w, 0)
    ref = oracle_linear(w, 0)
    assert torch.isfinite(out.float()).all()
    assert_out_close(out, ref, spec.act_dtype, f"{name} strong decay")


def test_denoise_is_bidirectional_readout():
    """All block rows read the block-end state: equal queries give equal rows."""
    spec = CASES["serving_batch64_r3"]
    w = gen(spec)
    install_states(w)
    blk = w.denoise[0]
    blk.q[:] = blk.q[:, :1].clone()
    out = run_linear(w).float()
    assert torch.allclose(out, out[:, :1].expand_as(out), atol=0, rtol=0)


def test_empty_batch_is_a_no_op():
    spec = CASES["tiny_fp32"]
    w = gen(spec)
    d = flare.linear_desc(0, spec.block_len, spec.num_qk_heads, spec.num_v_heads,
                          spec.head_dim_k, spec.head_dim_v, w.state_pool.shape[0],
                          flare.FLARE_DT_F32, 0.125)
    blk = w.denoise[0]
    out = torch.full_like(blk.v, 3.0)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert flare.flare_block_linear_attn(d, blk.q, blk.k, blk.v, blk.log_decay, blk.beta,
                                         w.state_pool, w.state_slot, out, st) == flare.FLARE_OK
    torch.cuda.synchronize()
    assert (out == 3.0).all()
