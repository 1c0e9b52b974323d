"""GPU parity of flare_short_conv (two-stream causal ShortConv of a block and
the commit of its conv state) against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import gen, status_word
from paper_2606_01774_gb300 import flare, workloads

pytestmark = pytest.mark.gpu
W = workloads.WORKLOADS
SC = W["shortconv_serving_batch64"]

CASES = {
    "w4_b32_r3": SC.replace(num_requests=3, prefix_lo=64, prefix_hi=128),
    "w4_b1": SC.replace(num_requests=4, block_len=1, prefix_lo=64, prefix_hi=128, seed=71),
    "w3_b7": SC.replace(num_requests=3, block_len=7, conv_width=3, prefix_lo=64, prefix_hi=128,
                        seed=72),
    "w2_b64": SC.replace(num_requests=2, block_len=64, conv_width=2, prefix_lo=64,
                         prefix_hi=128, seed=73),
    "w1_b16": SC.replace(num_requests=3, block_len=16, conv_width=1, prefix_lo=64,
                         prefix_hi=128, seed=74),
    "w4_fp32_small": W["tiny_fp32"].replace(num_requests=3, block_len=9, conv_width=4, seed=75),
    "w4_small_model": W["small_model_batch256"].replace(num_requests=5, conv_width=4, seed=76),
    # 120 channels: rows that do not tile by 512 bytes (one copy per row)
    "w4_c120": SC.replace(num_requests=3, block_len=11, num_qk_heads=1, num_v_heads=1,
                          head_dim_k=40, head_dim_v=40, prefix_lo=64, prefix_hi=128, seed=77),
}


# The ShortConv is a sum of W products in fp32 rounded once to the output type,
# so each element is within half a unit in the last place of the exact value
# plus the fp32 accumulation error: |gpu - exact| <= u |exact| with the unit
# roundoff u = 2^-8 (bf16, 8 significant bits) or 2^-24 (fp32), a few fp32
# roundings on top.  Outputs reach |y| ~ 10 (products of two normal
# variates), where a bf16 half-ulp is above the 2e-2 max-abs bound stated for
# the attention outputs, so the bound is relative.
REL = {"bf16": 2.0 ** -8 * 1.01, "f32": 2.0 ** -20}
ABS = 1e-6


def assert_rounded_close(gpu, ref, act_dtype, what=""):
    g = gpu.detach().double().cpu().numpy()
    assert np.isfinite(g).all(), f"{what}: non-finite GPU output"
    err = np.abs(g - ref)
    bound = REL[act_dtype] * np.abs(ref) + ABS
    worst = np.unravel_index(np.argmax(err - bound), err.shape)
    assert (err <= bound).all(), (f"{what}: |err| {err[worst]:.3e} > {bound[worst]:.3e} "
                                  f"at {worst}, ref {ref[worst]:.4f}")


def desc_of(spec, w, silu=True):
    act = flare.FLARE_DT_BF16 if spec.act_dtype == "bf16" else flare.FLARE_DT_F32
    return flare.conv_desc(spec.num_requests, spec.block_len, spec.conv_channels,
                           spec.conv_width, w.conv_state.shape[0], act,
                           flare.FLARE_ACT_SILU if silu else flare.FLARE_ACT_NONE)


def run_conv(spec, w, x, accept=None, silu=True, bias=True, expect_bits=0):
    out = torch.empty_like(x)
    st = status_word("cuda")
    rc = flare.flare_short_conv(desc_of(spec, w, silu), x, w.conv_state, w.state_slot,
                                w.conv_weight, w.conv_bias if bias else None, accept, out, st)
    flare.check(rc, "flare_short_conv")
    assert flare.flare_read_status(st)[1] == expect_bits
    return out


def oracle_conv(w, state_before, x, accept=None, silu=True, bias=True, requests=None):
    R = x.shape[0]
    req = list(range(R)) if requests is None else list(requests)
    i = torch.tensor(req, device="cuda")
    return oracle.short_conv(x[i].cpu(), state_before.cpu(), w.state_slot[i].cpu(),
                             w.conv_weight.cpu(), w.conv_bias.cpu() if bias else None,
                             silu=silu, accept_len=None if accept is None else accept[i].cpu())


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("silu,bias", [(True, True), (False, False)])
def test_shortconv_matches_oracle(name, silu, bias):
    spec = CASES[name]
    w = gen(spec)
    before = w.conv_state.clone()
    out = run_conv(spec, w, w.conv_x[0], silu=silu, bias=bias)
    ref = oracle_conv(w, before, w.conv_x[0], silu=silu, bias=bias)
    assert_rounded_close(out, ref["out"], spec.act_dtype, name)
    # the denoise call never writes the conv state
    assert torch.equal(w.conv_state.view(torch.uint8), before.view(torch.uint8))


@pytest.mark.parametrize("name", ["w4_b32_r3", "w3_b7", "w1_b16", "w4_fp32_small"])
def test_shortconv_commit_is_a_bit_copy(name):
    """Outputs of the state-update call and the committed state (the last W-1
    rows of old state ++ accepted rows) for n = 0, 1, W-2 and B; the state is
    copied bit for bit; unused (NaN) slots stay as they were."""
    spec = CASES[name]
    w = gen(spec)
    R, B, Wd = spec.num_requests, spec.block_len, spec.conv_width
    choices = [0, 1, max(Wd - 2, 0), B]
    acc = torch.tensor([choices[r % 4] for r in range(R)], dtype=torch.int32, device="cuda")
    acc.clamp_(0, B)
    before = w.conv_state.clone()
    out = run_conv(spec, w, w.conv_commit_x, accept=acc)
    ref = oracle_conv(w, before, w.conv_commit_x, accept=acc)
    assert_rounded_close(out, ref["out"], spec.act_dtype, name)
    slots = w.state_slot.long()
    got = w.conv_state[slots].double().cpu().numpy()
    np.testing.assert_array_equal(got, ref["state"])  # exact: a copy of representable values
    unused = torch.ones(w.conv_state.shape[0], dtype=torch.bool, device="cuda")
    unused[slots] = False
    assert torch.equal(w.conv_state[unused].view(torch.uint8), before[unused].view(torch.uint8))


def test_shortconv_full_size():
    """The full 64-request block in the launch configuration the bench times,
    every output against the oracle, then the commit at the full block."""
    spec = SC
    w = gen(spec)
    before = w.conv_state.clone()
    out = run_conv(spec, w, w.conv_x[0])
    ref = oracle_conv(w, before, w.conv_x[0])
    assert_rounded_close(out, ref["out"], spec.act_dtype, "shortconv full size")
    acc = torch.full((spec.num_requests,), spec.block_len, dtype=torch.int32, device="cuda")
    run_conv(spec, w, w.conv_commit_x, accept=acc)
    want = w.conv_commit_x[:, spec.block_len - (spec.conv_width - 1):]
    assert torch.equal(w.conv_state[w.state_slot.long()].view(torch.uint8),
                       want.contiguous().view(torch.uint8))


def test_shortconv_bad_slot_and_length_are_flagged():
    spec = CASES["w4_b32_r3"]
    w = gen(spec)
    before = w.conv_state.clone()
    acc = torch.tensor([0, spec.block_len + 1, 2], dtype=torch.int32, device="cuda")
    run_conv(spec, w, w.conv_commit_x, accept=acc, expect_bits=flare.FLARE_DEV_BAD_ACCEPT_LEN)
    assert torch.equal(w.conv_state[w.state_slot[1].long()].view(torch.uint8),
                       before[w.state_slot[1].long()].view(torch.uint8))
    w.state_slot[2] = w.conv_state.shape[0]
    run_conv(spec, w, w.conv_x[0], expect_bits=flare.FLARE_DEV_BAD_SLOT)


def test_shortconv_host_checks():
    spec = CASES["w4_b32_r3"]
    w = gen(spec)
    d = desc_of(spec, w)
    st = status_word("cuda")
    x = w.conv_x[0]
    out = torch.empty_like(x)
    d.width = 5
    assert flare.flare_short_conv(d, x, w.conv_state, w.state_slot, w.conv_weight, None, None,
                                  out, st) == flare.FLARE_ERR_UNSUPPORTED
    d.width = 4
    d.channels = 12
    assert flare.flare_short_conv(d, x, w.conv_state, w.state_slot, w.conv_weight, None, None,
                                  out, st) == flare.FLARE_ERR_UNSUPPORTED
    d.channels = spec.conv_channels
    assert flare.flare_short_conv(d, x, None, w.state_slot, w.conv_weight, None, None, out,
                                  st) == flare.FLARE_ERR_INVALID_ARGUMENT
