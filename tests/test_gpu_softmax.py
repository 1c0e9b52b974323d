"""GPU parity of flare_block_softmax_attn and the page indexing against the oracle."""
import math

import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import (assert_out_close, gen, oracle_softmax, reduced, run_softmax,
                         softmax_desc)
from paper_2606_01774_gb300 import flare, workloads

pytestmark = pytest.mark.gpu
W = workloads.WORKLOADS
LSE_ABS = 2e-3

CASES = {
    "tiny_fp32": W["tiny_fp32"],
    "single_request": W["single_request"],
    "serving_batch64_r3": reduced(W["serving_batch64"], 3, 512, 1500),
    "small_model_batch256_r4": reduced(W["small_model_batch256"], 4),
    "multistep_batch128_r3": reduced(W["multistep_batch128"], 3, 100, 900),
    "empty_and_short_prefix": W["serving_batch64"].replace(num_requests=4, prefix_lo=0,
                                                           prefix_hi=70, block_len=7, seed=41),
    "page16_d128": W["small_model_batch256"].replace(num_requests=3, page_size=16,
                                                     prefix_lo=1, prefix_hi=300, seed=42),
    # more work items than SMs, each a few tiles long and ending inside a page:
    # every CTA walks several items back to back, each with a zeroed partial tile
    "many_short_items_d128": W["small_model_batch256"].replace(num_requests=100, prefix_lo=1,
                                                               prefix_hi=200, seed=43),
    "many_short_items_d256": W["serving_batch64"].replace(num_requests=80, prefix_lo=1,
                                                          prefix_hi=300, seed=44),
}


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("mode", [flare.FLARE_MASK_BLOCK_BIDIR, flare.FLARE_MASK_BLOCK_CAUSAL])
def test_softmax_matches_oracle(name, mode):
    spec = CASES[name]
    w = gen(spec)
    out, lse = run_softmax(w, 0, mode)
    ref, ref_lse = oracle_softmax(w, 0, mode=mode)
    assert_out_close(out, ref, spec.act_dtype, f"{name} mode {mode}")
    assert np.abs(lse.double().cpu().numpy() - ref_lse).max() < LSE_ABS


@pytest.mark.parametrize("name", ["serving_batch64", "small_model_batch256", "multistep_batch128"])
def test_softmax_full_size_sampled(name):
    """Full batch in the launch configuration bench.py times; the oracle checks
    the shortest, the longest and one more request element by element."""
    spec = W[name]
    w = gen(spec)
    out, lse = run_softmax(w, spec.denoise_steps - 1)
    assert torch.isfinite(out).all()
    lens = w.prefix_len.cpu()
    sample = sorted({int(lens.argmin()), int(lens.argmax()), spec.num_requests // 2})
    ref, ref_lse = oracle_softmax(w, spec.denoise_steps - 1, sample)
    assert_out_close(out[sample], ref, spec.act_dtype, name)
    assert np.abs(lse[sample].double().cpu().numpy() - ref_lse).max() < LSE_ABS


@pytest.mark.parametrize("name", ["serving_batch64", "small_model_batch256"])
def test_softmax_full_size_every_request(name):
    """Full batch in the launch configuration bench.py times, every request,
    query head and block row element by element (outputs and log-sum-exp)."""
    spec = W[name]
    w = gen(spec)
    out, lse = run_softmax(w, spec.denoise_steps - 1)
    ref, ref_lse = oracle_softmax(w, spec.denoise_steps - 1)
    assert_out_close(out, ref, spec.act_dtype, name)
    assert np.abs(lse.double().cpu().numpy() - ref_lse).max() < LSE_ABS


def test_page_shuffle_is_bit_identical():
    """The same logical prefix stored at another permutation of physical pages
    gives bit-identical outputs (the paging is pure address arithmetic)."""
    spec = CASES["serving_batch64_r3"]
    w = gen(spec)
    out1, lse1 = run_softmax(w)
    n = w.k_pool.shape[0]
    g = torch.Generator(device="cuda")
    g.manual_seed(77)
    perm = torch.randperm(n, generator=g, device="cuda")
    k2 = torch.empty_like(w.k_pool)
    v2 = torch.empty_like(w.v_pool)
    k2[perm] = w.k_pool
    v2[perm] = w.v_pool
    tab = w.page_table.clone()
    used = tab >= 0
    tab[used] = perm[tab[used].long()].to(torch.int32)
    w.k_pool, w.v_pool, w.page_table = k2, v2, tab
    out2, lse2 = run_softmax(w)
    assert torch.equal(out1.view(torch.int16), out2.view(torch.int16))
    assert torch.equal(lse1.view(torch.int32), lse2.view(torch.int32))


@pytest.mark.parametrize("name", ["tiny_fp32", "serving_batch64_r3", "page16_d128"])
def test_debug_gather_is_bit_exact(name):
    spec = CASES[name]
    w = gen(spec)
    desc = softmax_desc(spec, w)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    for r in range(spec.num_requests):
        P = int(w.prefix_len[r])
        ko = torch.empty(P, spec.num_kv_heads, spec.head_dim, dtype=w.k_pool.dtype, device="cuda")
        vo = torch.empty_like(ko)
        flare.check(flare.flare_debug_gather_prefix(desc, w.k_pool, w.v_pool, w.page_table,
                                                    w.prefix_len, r, ko, vo, st))
        for pool, got in ((w.k_pool, ko), (w.v_pool, vo)):
            want = oracle.gather_prefix(r, pool.cpu(), w.page_table.cpu(), w.prefix_len.cpu(),
                                        spec.page_size)
            assert np.array_equal(got.double().cpu().numpy(), want)
    assert flare.flare_read_status(st) == (flare.FLARE_OK, 0)


def test_nan_poisoned_pool_does_not_leak():
    """Spare pages and the rows past each prefix end hold NaN; every output and
    lse must be finite."""
    spec = CASES["empty_and_short_prefix"]
    w = gen(spec)
    assert torch.isnan(w.k_pool.float()).any()
    for mode in (0, 1):
        out, lse = run_softmax(w, 0, mode)
        assert torch.isfinite(out.float()).all() and torch.isfinite(lse).all()


def test_more_requests_than_the_prepass_holds_on_chip():
    # 4100 requests: the validation pre-pass keeps the prefix lengths and the
    # bad requests of at most 4096 in shared memory, so this call takes its
    # global-memory path; one bad page on each side of that bound
    spec = W["tiny_fp32"].replace(name="many_requests", act_dtype="bf16", num_requests=4100,
                                  prefix_lo=1, prefix_hi=40, seed=45)
    w = gen(spec)
    bad = (5, 4099)
    for r in bad:
        w.page_table[r, 0] = w.k_pool.shape[0]
    sb = w.softmax[0]
    desc = softmax_desc(spec, w)
    nb = flare.flare_softmax_workspace_size(desc)
    ws = torch.empty(max(nb, 1), dtype=torch.uint8, device="cuda")
    out = torch.full_like(sb.q, 5.0)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    flare.check(flare.flare_block_softmax_attn(desc, sb.q, sb.k_blk, sb.v_blk, w.k_pool,
                                               w.v_pool, w.page_table, w.prefix_len, out, None,
                                               ws, nb, st))
    rc, bits = flare.flare_read_status(st)
    assert rc == flare.FLARE_ERR_DEVICE_STATUS and bits == flare.FLARE_DEV_BAD_PAGE
    for r in bad:
        assert (out[r] == 5.0).all()
    sample = [0, 6, 4095, 4096, 4098]
    ref, _ = oracle_softmax(w, 0, requests=sample)
    assert_out_close(out[sample], ref, spec.act_dtype, "many requests")
