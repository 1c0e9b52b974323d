"""GPU parity of the AR-Trust verify round against the oracle: the per-row
mask modes of flare_block_softmax_attn, flare_verify_linear_attn (token-causal
anchor/verify rows, bidirectional draft rows, cached verify states, live state
written in place) and flare_verify_commit (gather-scatter at the accepted
offset, all layers in one launch)."""
import math

import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import (assert_out_close, assert_states_close, gen, install_states,
                         linear_desc, oracle_softmax, oracle_verify, run_softmax,
                         run_verify_linear, status_word)
from paper_2606_01774_gb300 import flare, workloads

pytestmark = pytest.mark.gpu
W = workloads.WORKLOADS
V = W["ar_trust_verify_batch64"]
LSE_ABS = 2e-3

CASES = {
    # serving shapes (D = 256, G = 8, 31-row block) with shorter prefixes
    "verify_r3": V.replace(num_requests=3, prefix_lo=512, prefix_hi=1500),
    # small-model shapes (D = 128, G = 4), horizon 8 (15-row block)
    "verify_d128_n8": W["small_model_batch256"].replace(num_requests=5, block_len=15,
                                                        verify_horizon=8, seed=51),
    # the paper's mask figure: horizon 5 (9-row block), fp32 (CUDA-core softmax)
    "verify_fp32_n5": W["tiny_fp32"].replace(num_requests=3, block_len=9, verify_horizon=5,
                                             prefix_lo=20, prefix_hi=40, seed=52),
    # the longest block the kernels take: horizon 32, 63 rows
    "verify_n32": W["multistep_batch128"].replace(num_requests=3, prefix_lo=100, prefix_hi=900,
                                                  block_len=63, verify_horizon=32,
                                                  denoise_steps=1, accept="full", seed=53),
    # more work items than SMs, short prefixes ending inside a page
    "verify_many_short": V.replace(num_requests=80, prefix_lo=1, prefix_hi=300, seed=54),
}


def _max_verify(spec):
    return spec.verify_horizon - 1


# ---------------------------------------------------------------- softmax


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("mode", [flare.FLARE_MASK_ROW_TYPE_UNIFORM,
                                  flare.FLARE_MASK_ROW_TYPE_PER_REQUEST])
def test_row_type_softmax_matches_oracle(name, mode):
    spec = CASES[name]
    w = gen(spec)
    rt = w.row_type if mode == flare.FLARE_MASK_ROW_TYPE_PER_REQUEST else w.row_type[0].clone()
    out, lse = run_softmax(w, 0, mode, row_type=rt)
    ref, ref_lse = oracle_softmax(w, 0, mode=mode, row_type=rt)
    assert_out_close(out, ref, spec.act_dtype, f"{name} mode {mode}")
    assert np.abs(lse.double().cpu().numpy() - ref_lse).max() < LSE_ABS


@pytest.mark.parametrize("name", ["verify_r3", "verify_fp32_n5"])
def test_uniform_row_types_equal_the_block_modes(name):
    """All rows token-causal is the state-update mask and all rows
    bidirectional the denoise mask, bit for bit, in both encodings."""
    spec = CASES[name]
    w = gen(spec)
    R, B = spec.num_requests, spec.block_len
    for block_mode, rtype in ((flare.FLARE_MASK_BLOCK_CAUSAL, 0), (flare.FLARE_MASK_BLOCK_BIDIR, 1)):
        ref, ref_lse = run_softmax(w, 0, block_mode)
        for mode, shape in ((flare.FLARE_MASK_ROW_TYPE_UNIFORM, (B,)),
                            (flare.FLARE_MASK_ROW_TYPE_PER_REQUEST, (R, B))):
            rt = torch.full(shape, rtype, dtype=torch.uint8, device="cuda")
            out, lse = run_softmax(w, 0, mode, row_type=rt)
            assert torch.equal(out.view(torch.uint8), ref.view(torch.uint8))
            assert torch.equal(lse.view(torch.int32), ref_lse.view(torch.int32))


def test_row_type_softmax_full_size_sampled():
    """The full 64-request verify batch in the launch configuration the bench
    times; the oracle checks the shortest, the longest and one more request."""
    spec = V
    w = gen(spec)
    mode = flare.FLARE_MASK_ROW_TYPE_PER_REQUEST
    out, lse = run_softmax(w, 0, mode, row_type=w.row_type)
    assert torch.isfinite(out.float()).all()
    lens = w.prefix_len.cpu()
    sample = sorted({int(lens.argmin()), int(lens.argmax()), spec.num_requests // 2})
    ref, ref_lse = oracle_softmax(w, 0, sample, mode=mode, row_type=w.row_type)
    assert_out_close(out[sample], ref, spec.act_dtype, "verify full size")
    assert np.abs(lse[sample].double().cpu().numpy() - ref_lse).max() < LSE_ABS


def test_row_type_needs_a_pointer():
    spec = CASES["verify_r3"]
    w = gen(spec)
    desc = flare.softmax_desc(spec.num_requests, spec.block_len, spec.num_q_heads,
                              spec.num_kv_heads, spec.head_dim, spec.page_size,
                              w.k_pool.shape[0], w.page_table.shape[1], flare.FLARE_DT_BF16,
                              0.0625, flare.FLARE_MASK_ROW_TYPE_PER_REQUEST, None)
    sb = w.softmax[0]
    st = status_word("cuda")
    rc = flare.flare_block_softmax_attn(desc, sb.q, sb.k_blk, sb.v_blk, w.k_pool, w.v_pool,
                                        w.page_table, w.prefix_len, torch.empty_like(sb.q), None,
                                        None, 0, st)
    assert rc == flare.FLARE_ERR_INVALID_ARGUMENT


# ---------------------------------------------------------------- linear


def _check_verify(w, before, out, rec, max_verify, requests=None, verify_len=None):
    spec = w.spec
    req = list(range(spec.num_requests)) if requests is None else list(requests)
    vl = (w.verify_len if verify_len is None else verify_len).cpu()
    ref = oracle_verify(w, before, max_verify, req, verify_len)
    assert_out_close(out[req], ref["out"], spec.act_dtype, f"{spec.name} verify out")
    slots = w.state_slot.long()
    for n, r in enumerate(req):
        K = int(vl[r])
        if K:
            assert_states_close(rec[r, :K], ref["records"][n, :K], f"records r{r}")
        assert torch.isnan(rec[r, K:]).all(), "records past K were written"
        assert_states_close(w.state_pool[slots[r]][None], ref["state"][n][None], f"live r{r}")
    used = torch.zeros(w.state_pool.shape[0], dtype=torch.bool, device="cuda")
    used[slots] = True
    assert torch.equal(w.state_pool[~used].view(torch.int32), before[~used].view(torch.int32))


@pytest.mark.parametrize("name", list(CASES))
def test_verify_linear_matches_oracle(name):
    spec = CASES[name]
    w = gen(spec)
    install_states(w)
    before = w.state_pool.clone()
    mv = _max_verify(spec)
    out, rec = run_verify_linear(w, mv)
    _check_verify(w, before, out, rec, mv)


@pytest.mark.parametrize("which", ["cold_start", "all_verify"])
def test_verify_linear_extreme_lengths(which):
    """K = 0 for every request (cold start: only the anchor is token-causal,
    no state is cached) and K = L - 1 (every row token-causal, the live state
    is the block-end state)."""
    spec = CASES["verify_r3"]
    w = gen(spec)
    install_states(w)
    before = w.state_pool.clone()
    L = spec.block_len
    K = 0 if which == "cold_start" else L - 1
    vl = torch.full((spec.num_requests,), K, dtype=torch.int32, device="cuda")
    mv = max(K, 1)
    out, rec = run_verify_linear(w, mv, verify_len=vl)
    _check_verify(w, before, out, rec, mv, verify_len=vl)


def test_verify_linear_full_size_sampled():
    """The full 64-request batch in the launch configuration the bench times;
    oracle-built states for a sample of requests, the oracle checks those."""
    spec = V
    w = gen(spec)
    vl = w.verify_len.cpu()
    sample = sorted({int(vl.argmin()), int(vl.argmax()), spec.num_requests // 2})
    install_states(w, sample)
    before = w.state_pool.clone()
    mv = _max_verify(spec)
    out, rec = run_verify_linear(w, mv)
    assert torch.isfinite(out.float()).all()
    _check_verify(w, before, out, rec, mv, requests=sample)


def test_verify_bad_length_is_flagged_and_skipped():
    spec = CASES["verify_r3"]
    w = gen(spec)
    install_states(w)
    before = w.state_pool.clone()
    mv = _max_verify(spec)
    vl = w.verify_len.clone()
    vl[1] = mv + 1
    out, rec = run_verify_linear(w, mv, verify_len=vl, expect_bits=flare.FLARE_DEV_BAD_VERIFY_LEN)
    s1 = w.state_slot[1].long()
    assert torch.equal(w.state_pool[s1].view(torch.int32), before[s1].view(torch.int32))
    assert torch.isnan(rec[1]).all()
    _check_verify(w, before, out, rec, mv, requests=[0, 2], verify_len=vl)


# ---------------------------------------------------------------- commit


def test_verify_commit_restores_the_accepted_state():
    """Two layers in one launch: after the verify round and the commit every
    slot holds the cached state at the accepted offset bit for bit (a < K) or
    the verify round's live state (a = K), which is the replay of the anchor
    plus a drafts (path (a)) within the state tolerance; other slots keep
    their bits."""
    spec = CASES["verify_many_short"]
    layers = []
    for seed in (61, 62):
        w = gen(spec.replace(seed=seed))
        if layers:  # one slot per request, shared by every layer's pool
            w.state_slot = layers[0].state_slot.clone()
        install_states(w)
        layers.append(w)
    base = layers[0]
    vl, acc = base.verify_len, base.verify_accept
    mv = _max_verify(spec)
    runs = []
    for w in layers:
        before = w.state_pool.clone()
        _, rec = run_verify_linear(w, mv, verify_len=vl)
        runs.append((before, rec, w.state_pool.clone()))
    st = status_word("cuda")
    desc = linear_desc(spec, base.state_pool.shape[0])
    rc = flare.flare_verify_commit(desc, mv, [r[1] for r in runs], [w.state_pool for w in layers],
                                   base.state_slot, acc, vl, st)
    flare.check(rc, "flare_verify_commit")
    assert flare.flare_read_status(st) == (flare.FLARE_OK, 0)
    slots = base.state_slot.long()
    vl_c, acc_c = vl.cpu(), acc.cpu()
    for w, (before, rec, live) in zip(layers, runs):
        assert torch.equal(w.state_slot, base.state_slot)
        for r in range(spec.num_requests):
            a, K = int(acc_c[r]), int(vl_c[r])
            want = rec[r, a] if a < K else live[slots[r]]
            assert torch.equal(w.state_pool[slots[r]].view(torch.int32), want.view(torch.int32))
        used = torch.zeros(w.state_pool.shape[0], dtype=torch.bool, device="cuda")
        used[slots] = True
        assert torch.equal(w.state_pool[~used].view(torch.int32), live[~used].view(torch.int32))
        # path (a): replay the anchor and the accepted drafts with the oracle
        sample = list(range(0, spec.num_requests, 9))
        blk = w.denoise[0]
        i = torch.tensor(sample, device="cuda")
        o = oracle.gdr_per_token(None, blk.k[i].cpu(), blk.v[i].cpu(), blk.log_decay[i].cpu(),
                                 blk.beta[i].cpu(), before[slots[i]].cpu(),
                                 np.arange(len(sample), dtype=np.int32), (acc[i] + 1).cpu(),
                                 blockend=False)
        assert_states_close(w.state_pool[slots[i]], o["state"], "commit vs replay")


def test_verify_commit_bad_offset_is_flagged_and_skipped():
    spec = CASES["verify_r3"]
    w = gen(spec)
    install_states(w)
    mv = _max_verify(spec)
    _, rec = run_verify_linear(w, mv)
    live = w.state_pool.clone()
    acc = w.verify_len.clone()
    acc[0] = w.verify_len[0] + 1
    st = status_word("cuda")
    rc = flare.flare_verify_commit(linear_desc(spec, w.state_pool.shape[0]), mv, [rec],
                                   [w.state_pool], w.state_slot, acc, w.verify_len, st)
    flare.check(rc)
    _, bits = flare.flare_read_status(st)
    assert bits == flare.FLARE_DEV_BAD_VERIFY_LEN
    assert torch.equal(w.state_pool.view(torch.int32), live.view(torch.int32))
