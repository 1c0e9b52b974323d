"""Pins for the two-stream ShortConv part of the CPU oracle.

The read pattern is checked against the paper's ShortConv lag figure (which
stream and position each lag of a noisy output reads, in the interior of a
block, near its start, and with one-token blocks); the arithmetic against
torch's depthwise conv1d and SiLU in fp64 over the sequence (conv state ++
block); the state commit against its closed forms.
"""
import os

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _figure():
    rows = []
    for line in open(os.path.join(GOLDEN, "shortconv_lags_figure.txt")):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        head, reads = line.split(":")
        panel, B, start, pos = head.split()
        rows.append((panel, int(B), int(start), int(pos), reads.split()))
    return rows


@pytest.mark.parametrize("row", _figure(), ids=lambda r: r[0])
def test_lag_sources_match_the_paper_figure(row):
    """Tokens are one-hot on a channel of their own and w[c, i] = 10^i, so
    output channel c holds 10^i exactly when token c is read at lag i.  The
    serving-form inputs are built from the figure's setting: the block holds
    the noisy tokens of the output's block, the conv state the last W - 1 = 3
    clean tokens before the block's first position."""
    _, B, start, pos, want = row
    W = 4
    names = [f"c{p}" for p in range(start - W + 1, start)] + \
            [f"n{p}" for p in range(start, start + B)]
    C = len(names)
    ch = {n: i for i, n in enumerate(names)}
    x = np.zeros((1, B, C))
    for j in range(B):
        x[0, j, ch[f"n{start + j}"]] = 1.0
    state = np.zeros((1, W - 1, C))
    for j, p in enumerate(range(start - W + 1, start)):
        state[0, j, ch[f"c{p}"]] = 1.0
    weight = np.tile(10.0 ** np.arange(W), (C, 1))
    out = oracle.short_conv(x, state, np.array([0], np.int32), weight, silu=False)["out"]
    y = out[0, pos - start]
    got = [None] * W
    for c in range(C):
        if y[c] != 0.0:
            i = int(round(np.log10(y[c])))
            assert y[c] == 10.0 ** i
            got[i] = names[c]
    assert got == want


def _case(R=3, B=7, C=24, W=4, seed=0, nslots=5):
    g = np.random.default_rng(seed)
    x = g.standard_normal((R, B, C))
    state = g.standard_normal((nslots, W - 1, C))
    slot = g.permutation(nslots)[:R].astype(np.int32)
    weight = g.standard_normal((C, W)) * 0.5
    bias = g.standard_normal(C) * 0.1
    return x, state, slot, weight, bias


@pytest.mark.parametrize("W", [1, 2, 3, 4])
@pytest.mark.parametrize("silu", [False, True])
def test_matches_torch_depthwise_conv1d(W, silu):
    """Library routine: torch conv1d (groups = C, fp64) over the sequence
    conv state ++ block, without padding, then SiLU."""
    x, state, slot, weight, bias = _case(W=W, seed=W)
    out = oracle.short_conv(x, state, slot, weight, bias, silu=silu)["out"]
    R, B, C = x.shape
    for r in range(R):
        seq = np.concatenate([state[slot[r]], x[r]], 0)  # [W-1+B, C]
        inp = torch.tensor(seq.T[None])                   # [1, C, W-1+B]
        ker = torch.tensor(weight[:, ::-1].copy()[:, None, :])  # tap k multiplies lag W-1-k
        y = torch.nn.functional.conv1d(inp, ker, torch.tensor(bias), groups=C)[0].T
        if silu:
            y = torch.nn.functional.silu(y)
        np.testing.assert_allclose(out[r], y.numpy(), rtol=1e-13, atol=1e-13)


def test_width_one_is_pointwise():
    x, state, slot, weight, bias = _case(W=1, seed=9)
    out = oracle.short_conv(x, state, slot, weight, bias, silu=False)["out"]
    np.testing.assert_allclose(out, bias + weight[:, 0] * x, rtol=1e-14, atol=1e-14)


@pytest.mark.parametrize("W", [1, 2, 4])
def test_state_commit_closed_forms(W):
    """n = 0 keeps the old state; n >= W - 1 keeps the last W - 1 accepted rows;
    0 < n < W - 1 shifts the old state left by n and appends the n rows."""
    R, B = 4, 6
    x, state, slot, weight, bias = _case(R=R, B=B, W=W, seed=20 + W, nslots=6)
    acc = np.array([0, 1, B, min(2, B)], np.int32)
    st = oracle.short_conv(x, state, slot, weight, bias, accept_len=acc)["state"]
    for r in range(R):
        n, old = int(acc[r]), state[slot[r]]
        if W == 1:
            assert st[r].shape == (0, x.shape[2])
        elif n == 0:
            np.testing.assert_array_equal(st[r], old)
        elif n >= W - 1:
            np.testing.assert_array_equal(st[r], x[r, n - (W - 1):n])
        else:
            np.testing.assert_array_equal(st[r], np.concatenate([old[n:], x[r, :n]], 0))


def test_commit_then_next_block_equals_one_long_sequence():
    """Committing a block and convolving the next one from the new state
    equals convolving the two blocks as one sequence from the old state."""
    x, state, slot, weight, bias = _case(R=2, B=10, W=4, seed=31)
    B1 = 6
    acc = np.full(2, B1, np.int32)
    a = oracle.short_conv(x[:, :B1], state, slot, weight, bias, accept_len=acc)
    pool2 = state.copy()
    pool2[slot] = a["state"]
    b = oracle.short_conv(x[:, B1:], pool2, slot, weight, bias)
    whole = oracle.short_conv(x, state, slot, weight, bias)["out"]
    np.testing.assert_allclose(np.concatenate([a["out"], b["out"]], 1), whole, atol=1e-14)


def test_bad_arguments_rejected():
    x, state, slot, weight, bias = _case()
    with pytest.raises(ValueError):
        oracle.short_conv(x, state, np.array([0, 1, 9], np.int32), weight, bias)
    with pytest.raises(ValueError):
        oracle.short_conv(x, state, slot, weight, bias, accept_len=np.array([0, 8, 1], np.int32))
