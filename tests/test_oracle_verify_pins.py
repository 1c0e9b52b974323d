"""Pins for the AR-Trust verify-round part of the CPU oracle.

Each check compares the oracle with something other than itself: the attention
pattern printed in the paper's AR-Trust mask figure, torch's fp64
scaled_dot_product_attention on a densely assembled masked problem, the
paper's statement that replaying the accepted updates (path (a)) and caching
then scattering (path (b)) give the same state, and closed forms of the gated
delta rule (pure decay; unit steps on basis keys that overwrite state rows).
"""
import math
import os

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _unit(x):
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


def _read_figure():
    rows, types = [], None
    for line in open(os.path.join(GOLDEN, "ar_trust_mask_figure.txt")):
        line = line.strip()
        if line.startswith("# row_types"):
            types = [int(x) for x in line.split(":")[1].split()]
        elif line and not line.startswith("#"):
            rows.append([c == "1" for c in line])
    return np.array(rows, bool), np.array(types, np.uint8)


def _layout_types(L, K):
    """Row types of the verify-round block layout: anchor and K verify rows
    token-causal (0), everything after them bidirectional (1)."""
    t = np.ones(L, np.uint8)
    t[:K + 1] = 0
    return t


def _one_hot_case(P, B, D):
    """q = 0 and one-hot values: the output of row t is the indicator of its
    visible keys divided by their count, so the mask can be read off."""
    p = 8
    npg = -(-P // p) if P else 0
    kp = np.zeros((max(npg, 1) + 1, 1, p, D))
    vp = np.zeros_like(kp)
    table = np.zeros((1, max(npg, 1)), np.int32)
    for j in range(P):
        table[0, j // p] = j // p + 1  # page 0 stays unused
        vp[j // p + 1, 0, j % p, j] = 1.0
    vb = np.zeros((1, B, 1, D))
    for i in range(B):
        vb[0, i, 0, P + i] = 1.0
    q = np.zeros((1, B, 1, D))
    kb = np.zeros((1, B, 1, D))
    return q, kb, vb, kp, vp, table, np.array([P], np.int32)


@pytest.mark.parametrize("mode", [2, 3])
def test_row_type_mask_matches_paper_figure(mode):
    fig, types = _read_figure()
    B, P = len(types), fig.shape[1] - len(types)
    q, kb, vb, kp, vp, table, lens = _one_hot_case(P, B, fig.shape[1])
    rt = types if mode == 2 else types[None]
    out, _ = oracle.block_softmax(q, kb, vb, kp, vp, table, lens, scale=1.0, mask_mode=mode,
                                  row_type=rt)
    seen = out[0, :, 0] > 0
    np.testing.assert_array_equal(seen, fig)
    np.testing.assert_allclose(out[0, :, 0].sum(1), 1.0, atol=1e-14)


def test_row_types_reduce_to_the_two_uniform_modes():
    """All-causal row types are the state-update mask, all-bidirectional ones
    the denoise mask, in both compact encodings."""
    fig, types = _read_figure()
    B, P = len(types), fig.shape[1] - len(types)
    q, kb, vb, kp, vp, table, lens = _one_hot_case(P, B, fig.shape[1])
    for mode_uniform, rtype in ((1, 0), (0, 1)):
        ref, _ = oracle.block_softmax(q, kb, vb, kp, vp, table, lens, mask_mode=mode_uniform)
        for mode in (2, 3):
            rt = np.full(B if mode == 2 else (1, B), rtype, np.uint8)
            out, _ = oracle.block_softmax(q, kb, vb, kp, vp, table, lens, mask_mode=mode,
                                          row_type=rt)
            np.testing.assert_array_equal(out > 0, ref > 0)


def _paged(R, B, Hq, Hkv, D, p, lens, seed):
    g = np.random.default_rng(seed)
    dk = [g.standard_normal((P, Hkv, D)) for P in lens]
    dvv = [g.standard_normal((P, Hkv, D)) for P in lens]
    npages = [-(-P // p) for P in lens]
    num_pages = sum(npages) + 2
    ids = g.permutation(num_pages)
    kp = np.full((num_pages, Hkv, p, D), np.nan)
    vp = kp.copy()
    table = np.zeros((R, max(max(npages), 1)), np.int32)
    off = 0
    for r, P in enumerate(lens):
        for j in range(P):
            if j % p == 0:
                table[r, j // p] = ids[off]
                off += 1
            kp[table[r, j // p], :, j % p] = dk[r][j]
            vp[table[r, j // p], :, j % p] = dvv[r][j]
    q = g.standard_normal((R, B, Hq, D))
    kb = g.standard_normal((R, B, Hkv, D))
    vb = g.standard_normal((R, B, Hkv, D))
    return q, kb, vb, kp, vp, table, np.array(lens, np.int32), dk, dvv


def test_per_request_row_types_match_library_sdpa():
    """Per-request layouts (cold start K = 0, partial and full verify) against
    torch's fp64 SDPA over the densely assembled visible set."""
    R, B, Hq, Hkv, D, p = 3, 7, 4, 2, 16, 4
    lens = (5, 0, 11)
    Ks = (0, 3, 6)
    q, kb, vb, kp, vp, table, lens_a, dk, dvv = _paged(R, B, Hq, Hkv, D, p, lens, seed=5)
    rt = np.stack([_layout_types(B, K) for K in Ks])
    out, lse = oracle.block_softmax(q, kb, vb, kp, vp, table, lens_a, mask_mode=3, row_type=rt)
    G = Hq // Hkv
    for r in range(R):
        P = lens[r]
        Kd = np.concatenate([dk[r], kb[r]], 0)
        Vd = np.concatenate([dvv[r], vb[r]], 0)
        mask = np.ones((B, P + B), bool)
        for t in range(B):
            if rt[r, t] == 0:
                mask[t, P + t + 1:] = False
        for h in range(Hq):
            want = torch.nn.functional.scaled_dot_product_attention(
                torch.tensor(q[r, :, h])[None, None], torch.tensor(Kd[:, h // G])[None, None],
                torch.tensor(Vd[:, h // G])[None, None],
                attn_mask=torch.tensor(mask)[None, None])[0, 0].numpy()
            np.testing.assert_allclose(out[r, :, h], want, atol=1e-12)
            z = np.where(mask, q[r, :, h] @ Kd[:, h // G].T / math.sqrt(D), -np.inf)
            m = z.max(1)
            np.testing.assert_allclose(lse[r, :, h], m + np.log(np.exp(z - m[:, None]).sum(1)),
                                       atol=1e-12)


def test_row_type_values_are_checked():
    q, kb, vb, kp, vp, table, lens = _one_hot_case(3, 4, 8)
    with pytest.raises(ValueError):
        oracle.block_softmax(q, kb, vb, kp, vp, table, lens, mask_mode=2,
                             row_type=np.array([0, 2, 1, 1], np.uint8))
    with pytest.raises(ValueError):
        oracle.block_softmax(q, kb, vb, kp, vp, table, lens, mask_mode=3,
                             row_type=np.zeros(4, np.uint8))


# ---------------------------------------------------------------- gated delta rule


def _verify_case(R=3, L=9, Hk=2, Hv=4, dk=16, dv=8, Ks=(0, 3, 8), max_verify=8, seed=0):
    g = np.random.default_rng(seed)
    q = _unit(g.standard_normal((R, L, Hk, dk)))
    k = _unit(g.standard_normal((R, L, Hk, dk)))
    v = g.standard_normal((R, L, Hv, dv))
    ld = -np.log1p(np.exp(g.standard_normal((R, L, Hv))))
    beta = 1.0 / (1.0 + np.exp(-g.standard_normal((R, L, Hv))))
    pool = g.standard_normal((R + 2, Hv, dk, dv)) * 0.3
    slot = g.permutation(R + 2)[:R].astype(np.int32)
    return q, k, v, ld, beta, pool, slot, np.array(Ks, np.int32), max_verify


def test_verify_cache_equals_replay():
    """Path (b) (cache S^(t) during the verify forward) equals path (a)
    (replay the accepted updates): every cached state, the live state, and the
    two readouts agree with the commit / causal / block-end forms."""
    q, k, v, ld, beta, pool, slot, Ks, mv = _verify_case()
    R, L = q.shape[:2]
    o = oracle.gdr_verify(q, k, v, ld, beta, pool, slot, Ks, mv)
    full = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot, causal=True)
    for r in range(R):
        K = int(Ks[r])
        for t in range(K):
            st = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot,
                                      np.full(R, t + 1, np.int32))["state"]
            np.testing.assert_allclose(o["records"][r, t], st[r], rtol=1e-12, atol=1e-12)
        st = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot,
                                  np.full(R, K + 1, np.int32))["state"]
        np.testing.assert_allclose(o["state"][r], st[r], rtol=1e-12, atol=1e-12)
        np.testing.assert_array_equal(o["records"][r, K:], 0.0)
        np.testing.assert_allclose(o["out"][r, :K + 1], full["causal"][r, :K + 1], atol=1e-12)
        np.testing.assert_allclose(o["out"][r, K + 1:], full["blockend"][r, K + 1:], atol=1e-12)


def test_verify_pure_decay_closed_form():
    """beta = 0: every state is exp(sum of the log-gates so far) S0."""
    q, k, v, ld, beta, pool, slot, Ks, mv = _verify_case(seed=1)
    beta = np.zeros_like(beta)
    o = oracle.gdr_verify(q, k, v, ld, beta, pool, slot, Ks, mv)
    R, L, Hv = ld.shape
    Hk = q.shape[2]
    s = 1.0 / math.sqrt(q.shape[3])
    for r in range(R):
        K = int(Ks[r])
        cum = np.cumsum(ld[r], axis=0)  # [L, Hv]
        S0 = pool[slot[r]]
        for t in range(K):
            np.testing.assert_allclose(o["records"][r, t], np.exp(cum[t])[:, None, None] * S0,
                                       rtol=1e-13)
        np.testing.assert_allclose(o["state"][r], np.exp(cum[K])[:, None, None] * S0, rtol=1e-13)
        for t in range(L):
            gt = cum[t] if t <= K else cum[L - 1]
            for j in range(Hv):
                want = s * math.exp(gt[j]) * S0[j].T @ q[r, t, j * Hk // Hv]
                np.testing.assert_allclose(o["out"][r, t, j], want, rtol=1e-12, atol=1e-14)


def test_verify_basis_keys_overwrite_rows():
    """g = 0, beta = 1, k_t = e_{pi(t)}: token t overwrites state row pi(t)
    with v_t, so S^(t) is S0 with rows pi(0..t) replaced."""
    R, L, Hk, Hv, dk, dv = 2, 6, 1, 2, 8, 5
    g = np.random.default_rng(7)
    perm = g.permutation(dk)[:L]
    k = np.zeros((R, L, Hk, dk))
    for t in range(L):
        k[:, t, :, perm[t]] = 1.0
    q = g.standard_normal((R, L, Hk, dk))
    v = g.standard_normal((R, L, Hv, dv))
    ld = np.zeros((R, L, Hv))
    beta = np.ones((R, L, Hv))
    pool = g.standard_normal((R, Hv, dk, dv))
    slot = np.arange(R, dtype=np.int32)
    Ks = np.array([4, 2], np.int32)
    o = oracle.gdr_verify(q, k, v, ld, beta, pool, slot, Ks, 5)
    for r in range(R):
        S = pool[r].copy()
        for t in range(L):
            S[:, perm[t], :] = v[r, t]
            if t < Ks[r]:
                np.testing.assert_allclose(o["records"][r, t], S, atol=1e-14)
            if t == Ks[r]:
                np.testing.assert_allclose(o["state"][r], S, atol=1e-14)


def test_verify_rejects_bad_lengths():
    q, k, v, ld, beta, pool, slot, Ks, mv = _verify_case()
    for bad, m in ((np.array([0, 3, 9], np.int32), 9), (np.array([0, 3, 8], np.int32), 7),
                   (np.array([-1, 3, 8], np.int32), 8)):
        with pytest.raises(ValueError):
            oracle.gdr_verify(q, k, v, ld, beta, pool, slot, bad, m)


def test_verify_commit_gather_scatter():
    """Brute force on a tiny case: after the verify round and the commit with
    accepted offset a, each layer's slot holds the state of replaying the
    anchor plus a drafts (path (a)); a = K leaves the slot as the verify round
    left it; slots not named stay bit-identical."""
    q, k, v, ld, beta, pool, slot, Ks, mv = _verify_case(R=3, Ks=(0, 3, 8), seed=3)
    R = q.shape[0]
    layers = []
    for layer in range(2):
        ll = ld + 0.1 * layer
        o = oracle.gdr_verify(q, k, v, ll, beta, pool, slot, Ks, mv)
        live = pool.copy()
        live[slot] = o["state"]
        layers.append((ll, o, live))
    acc = np.array([0, 1, 8], np.int32)
    new = oracle.verify_commit([x[1]["records"] for x in layers], [x[2] for x in layers], slot,
                               acc, Ks)
    for (ll, o, live), got in zip(layers, new):
        replay = oracle.gdr_per_token(q, k, v, ll, beta, pool, slot, acc + 1)["state"]
        for r in range(R):
            np.testing.assert_allclose(got[slot[r]], replay[r], rtol=1e-12, atol=1e-12)
            if acc[r] == Ks[r]:
                np.testing.assert_array_equal(got[slot[r]], live[slot[r]])
        others = np.setdiff1d(np.arange(pool.shape[0]), slot)
        np.testing.assert_array_equal(got[others], live[others])
    with pytest.raises(ValueError):
        oracle.verify_commit([layers[0][1]["records"]], [layers[0][2]], slot,
                             np.array([0, 4, 8], np.int32), Ks)
