"""Pins for the CPU oracle: checks against what the paper and the mathematics fix.

None of these compares the oracle with itself.  Each pin is a worked example
derived by hand, a closed form, an invariant the paper states, a second
algorithm for the same quantity, or a library routine on a special case, and
each is chosen so that a plausible slip in the oracle (a dropped gate, a sign,
a transposed state, a causal instead of block-end readout, a wrong head or page
index) fails at least one of them.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(1234)


def _unit(x):
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


def _random_gdr(R=2, B=8, Hk=2, Hv=4, dk=16, dv=24, nslots=None, seed=0):
    g = np.random.default_rng(seed)
    nslots = nslots or R + 2
    q = _unit(g.standard_normal((R, B, Hk, dk)))
    k = _unit(g.standard_normal((R, B, Hk, dk)))
    v = g.standard_normal((R, B, Hv, dv))
    ld = -np.log1p(np.exp(g.standard_normal((R, B, Hv))))
    beta = 1.0 / (1.0 + np.exp(-g.standard_normal((R, B, Hv))))
    pool = g.standard_normal((nslots, Hv, dk, dv)) * 0.3
    slot = g.permutation(nslots)[:R].astype(np.int32)
    return q, k, v, ld, beta, pool, slot


# ---------------------------------------------------------------- gated delta rule


def test_gdr_worked_example_by_hand():
    """Hand-derived 2x2 example (tests/golden/gdr_worked_2x2.json)."""
    gx = json.load(open(os.path.join(GOLDEN, "gdr_worked_2x2.json")))
    k = np.array(gx["k"])[None, :, None, :]
    q = np.array(gx["q"])[None, :, None, :]
    v = np.array(gx["v"])[None, :, None, :]
    ld = np.log(np.array(gx["alpha"]))[None, :, None]
    beta = np.array(gx["beta"])[None, :, None]
    pool = np.array(gx["S0"])[None, None]
    slot = np.array([0], np.int32)
    ex = gx["expect"]
    for r in (0, 1, 2):
        o = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot, np.array([r], np.int32),
                                 scale=gx["scale"], causal=True)
        np.testing.assert_allclose(o["state"][0, 0], ex[f"state_r{r}"], atol=1e-13)
        np.testing.assert_allclose(o["causal"][0, :, 0], ex["causal"], atol=1e-13)
        np.testing.assert_allclose(o["blockend"][0, :, 0], ex["blockend"], atol=1e-13)
        c = oracle.gdr_chunked(q, k, v, ld, beta, pool, slot, np.array([r], np.int32),
                               scale=gx["scale"])
        np.testing.assert_allclose(c["state"][0, 0], ex[f"state_r{r}"], atol=1e-13)
        np.testing.assert_allclose(c["blockend"][0, :, 0], ex["blockend"], atol=1e-13)


@pytest.mark.parametrize("B", [1, 8, 13, 64])
def test_per_token_equals_chunkwise(B):
    """Eq. per-step-fwd run token by token equals the chunkwise WY/UT form
    (Eq. chunk-state / Eq. f-blk); the paper uses the two interchangeably."""
    q, k, v, ld, beta, pool, slot = _random_gdr(B=B, seed=B)
    for acc in (np.array([B, 0], np.int32), np.array([max(B // 2, 1), B], np.int32)):
        a = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot, acc)
        b = oracle.gdr_chunked(q, k, v, ld, beta, pool, slot, acc)
        for key in ("blockend", "state"):
            err = np.linalg.norm(a[key] - b[key]) / np.linalg.norm(b[key])
            assert err < 1e-10, (key, err)


def test_matches_compact_recurrence():
    """Eq. gdn-recurrence in its compact matrix form
    S_t = alpha_t (I - beta_t k_t k_t^T) S_{t-1} + beta_t k_t v_t^T."""
    q, k, v, ld, beta, pool, slot = _random_gdr(R=1, B=6, Hk=1, Hv=1, dk=5, dv=3, seed=7)
    S = pool[slot[0], 0].copy()
    states = []
    for t in range(6):
        kt = k[0, t, 0][:, None]
        S = math.exp(ld[0, t, 0]) * (np.eye(5) - beta[0, t, 0] * kt @ kt.T) @ S \
            + beta[0, t, 0] * kt @ v[0, t, 0][None, :]
        states.append(S.copy())
    for r in range(7):
        o = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot, np.array([r], np.int32),
                                 causal=True)
        want = pool[slot[0], 0] if r == 0 else states[r - 1]
        np.testing.assert_allclose(o["state"][0, 0], want, rtol=1e-12, atol=1e-13)
    s = 1 / math.sqrt(5)
    for t in range(6):
        np.testing.assert_allclose(o["causal"][0, t, 0], s * states[t].T @ q[0, t, 0], atol=1e-13)
        np.testing.assert_allclose(o["blockend"][0, t, 0], s * states[-1].T @ q[0, t, 0],
                                   atol=1e-13)


def test_beta_zero_is_pure_decay():
    """beta = 0: S_r = exp(sum_{i<=r} g_i) S0 and o~_l = s exp(sum_B g) S0^T q_l."""
    q, k, v, ld, beta, pool, slot = _random_gdr(seed=3)
    beta[:] = 0.0
    acc = np.array([3, 8], np.int32)
    for fn in (oracle.gdr_per_token, oracle.gdr_chunked):
        o = fn(q, k, v, ld, beta, pool, slot, acc)
        for r in range(2):
            for j in range(4):
                S0 = pool[slot[r], j]
                want = math.exp(ld[r, :acc[r], j].sum()) * S0
                np.testing.assert_allclose(o["state"][r, j], want, rtol=1e-12)
                h = j * 2 // 4
                for l in range(8):
                    wo = math.exp(ld[r, :, j].sum()) * S0.T @ q[r, l, h] / 4.0
                    np.testing.assert_allclose(o["blockend"][r, l, j], wo, rtol=1e-11, atol=1e-14)


def test_basis_keys_replace_rows():
    """g = 0, beta = 1, k_t = e_{pi(t)}: each step overwrites row pi(t) of S
    with v_t (the delta rule's exact replacement); the last write wins."""
    dk, dv, B = 8, 5, 6
    pi = [3, 1, 3, 6, 0, 1]
    k = np.zeros((1, B, 1, dk))
    for t, i in enumerate(pi):
        k[0, t, 0, i] = 1.0
    v = rng.standard_normal((1, B, 1, dv))
    q = rng.standard_normal((1, B, 1, dk))
    ld = np.zeros((1, B, 1))
    beta = np.ones((1, B, 1))
    pool = rng.standard_normal((1, 1, dk, dv))
    slot = np.array([0], np.int32)
    for r in range(B + 1):
        want = pool[0, 0].copy()
        for t in range(r):
            want[pi[t]] = v[0, t, 0]
        for fn in (oracle.gdr_per_token, oracle.gdr_chunked):
            o = fn(q, k, v, ld, beta, pool, slot, np.array([r], np.int32), scale=1.0)
            np.testing.assert_allclose(o["state"][0, 0], want, atol=1e-14)
            if r == B:
                np.testing.assert_allclose(o["blockend"][0, :, 0], q[0, :, 0] @ want, atol=1e-13)


def test_single_token_from_zero_state():
    """S0 = 0, B = 1: S_1 = beta k v^T and o = s beta (q . k) v."""
    q, k, v, ld, beta, pool, slot = _random_gdr(R=1, B=1, Hk=1, Hv=1, dk=7, dv=4, seed=5)
    pool[:] = 0.0
    o = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot, None, scale=0.25, causal=True)
    np.testing.assert_allclose(o["state"][0, 0], beta[0, 0, 0] * np.outer(k[0, 0, 0], v[0, 0, 0]),
                               atol=1e-15)
    want = 0.25 * beta[0, 0, 0] * (q[0, 0, 0] @ k[0, 0, 0]) * v[0, 0, 0]
    np.testing.assert_allclose(o["blockend"][0, 0, 0], want, atol=1e-15)
    np.testing.assert_allclose(o["causal"][0, 0, 0], want, atol=1e-15)


def test_unit_step_memorises_value():
    """beta = 1, g = 0, |k| = 1: after step t the state returns v_t at key k_t
    (S_t^T k_t = v_t), so the causal readout with q_t = k_t is s v_t."""
    q, k, v, ld, beta, pool, slot = _random_gdr(R=1, B=5, Hk=1, Hv=1, dk=9, dv=4, seed=11)
    ld[:] = 0.0
    beta[:] = 1.0
    q = k.copy()
    o = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot, None, scale=1.0, causal=True)
    np.testing.assert_allclose(o["causal"][0, :, 0], v[0, :, 0], atol=1e-13)


def test_blockend_readout_is_bidirectional():
    """Every block row reads the same block-end state (Eq. noisy-block-fwd):
    identical queries give identical outputs at every position, which a
    token-causal readout would not."""
    q, k, v, ld, beta, pool, slot = _random_gdr(R=1, B=6, seed=2)
    q[:] = q[:, :1]
    o = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot, None, causal=True)
    for l in range(6):
        np.testing.assert_allclose(o["blockend"][0, l], o["blockend"][0, 5], atol=1e-15)
    np.testing.assert_allclose(o["causal"][0, 5], o["blockend"][0, 5], atol=1e-15)
    assert np.abs(o["causal"][0, 0] - o["blockend"][0, 0]).max() > 1e-3


def test_accept_zero_leaves_state_unchanged():
    q, k, v, ld, beta, pool, slot = _random_gdr(seed=9)
    o = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot, np.zeros(2, np.int32))
    assert np.array_equal(o["state"], pool[slot])


def test_grouped_value_heads_read_their_qk_head():
    """With Hv = 2 Hk, value head j reads q/k head j // 2: equal to a run whose
    q/k heads are duplicated explicitly."""
    q, k, v, ld, beta, pool, slot = _random_gdr(Hk=2, Hv=4, seed=4)
    a = oracle.gdr_per_token(q, k, v, ld, beta, pool, slot, None, causal=True)
    rep = [0, 0, 1, 1]
    b = oracle.gdr_per_token(q[:, :, rep], k[:, :, rep], v, ld, beta, pool, slot, None,
                             causal=True)
    for key in a:
        np.testing.assert_allclose(a[key], b[key], atol=1e-15)
    # and not the other grouping
    c = oracle.gdr_per_token(q[:, :, [0, 1, 0, 1]], k[:, :, [0, 1, 0, 1]], v, ld, beta, pool,
                             slot, None)
    assert np.abs(c["blockend"] - a["blockend"]).max() > 1e-3


def test_bf16_inputs_widen_exactly():
    q, k, v, ld, beta, pool, slot = _random_gdr(seed=6)
    qb, kb, vb = (torch.tensor(x, dtype=torch.bfloat16) for x in (q, k, v))
    a = oracle.gdr_per_token(qb, kb, vb, ld.astype(np.float32), beta.astype(np.float32),
                             pool.astype(np.float32), slot)
    b = oracle.gdr_per_token(qb.double().numpy(), kb.double().numpy(), vb.double().numpy(),
                             ld.astype(np.float32).astype(np.float64),
                             beta.astype(np.float32).astype(np.float64),
                             pool.astype(np.float32).astype(np.float64), slot)
    for key in a:
        assert np.array_equal(a[key], b[key])


def test_invalid_slot_and_accept_rejected():
    q, k, v, ld, beta, pool, slot = _random_gdr(seed=8)
    with pytest.raises(ValueError):
        oracle.gdr_per_token(q, k, v, ld, beta, pool, np.array([0, 99], np.int32))
    with pytest.raises(ValueError):
        oracle.gdr_per_token(q, k, v, ld, beta, pool, slot, np.array([9, 1], np.int32))


# ---------------------------------------------------------------- softmax


def _paged_case(R=3, B=4, Hq=4, Hkv=2, D=16, p=4, lens=(0, 5, 12), seed=0, poison=True):
    """Build a paged pool from dense per-request prefixes with a python scatter
    loop written here (independent of the oracle's gather)."""
    g = np.random.default_rng(seed)
    dense_k = [g.standard_normal((P, Hkv, D)) for P in lens]
    dense_v = [g.standard_normal((P, Hkv, D)) for P in lens]
    npages = [-(-P // p) for P in lens]
    max_pages = max(max(npages), 1)
    num_pages = sum(npages) + 3
    ids = g.permutation(num_pages)
    kp = np.full((num_pages, Hkv, p, D), np.nan if poison else 0.0)
    vp = kp.copy()
    table = -np.ones((R, max_pages), np.int32)
    off = 0
    for r, P in enumerate(lens):
        for j in range(P):
            if j % p == 0:
                table[r, j // p] = ids[off]
                off += 1
            page = table[r, j // p]
            kp[page, :, j % p] = dense_k[r][j]
            vp[page, :, j % p] = dense_v[r][j]
    q = g.standard_normal((R, B, Hq, D))
    kb = g.standard_normal((R, B, Hkv, D))
    vb = g.standard_normal((R, B, Hkv, D))
    return dict(q=q, kb=kb, vb=vb, kp=kp, vp=vp, table=table, lens=np.array(lens, np.int32),
                dense_k=dense_k, dense_v=dense_v, p=p)


def test_softmax_worked_example_by_hand():
    gx = json.load(open(os.path.join(GOLDEN, "softmax_worked.json")))
    kp = np.full((2, 1, 2, 2), np.nan)
    vp = np.full((2, 1, 2, 2), np.nan)
    kp[1, 0] = gx["prefix_k"]
    vp[1, 0] = gx["prefix_v"]
    q = np.array(gx["q"])[None, :, None, :]
    kb = np.array(gx["block_k"])[None, :, None, :]
    vb = np.array(gx["block_v"])[None, :, None, :]
    ex = gx["expect"]
    for mode, tag in ((0, "bidir"), (1, "causal")):
        out, lse = oracle.block_softmax(q, kb, vb, kp, vp, gx["page_table"], gx["prefix_len"],
                                        scale=1.0, mask_mode=mode)
        np.testing.assert_allclose(out[0, :, 0], ex[f"{tag}_out"], atol=1e-14)
        np.testing.assert_allclose(lse[0, :, 0], ex[f"{tag}_lse"], atol=1e-14)


@pytest.mark.parametrize("mode", [0, 1])
def test_softmax_matches_library_sdpa(mode):
    """Special case that reduces to a library routine: torch's fp64
    scaled_dot_product_attention over the densely assembled visible set."""
    c = _paged_case()
    out, lse = oracle.block_softmax(c["q"], c["kb"], c["vb"], c["kp"], c["vp"], c["table"],
                                    c["lens"], mask_mode=mode)
    R, B, Hq, D = c["q"].shape
    G = Hq // c["kb"].shape[2]
    for r in range(R):
        P = int(c["lens"][r])
        K = np.concatenate([c["dense_k"][r], c["kb"][r]], 0)  # [P+B, Hkv, D]
        V = np.concatenate([c["dense_v"][r], c["vb"][r]], 0)
        mask = np.ones((B, P + B), bool)
        if mode == 1:
            mask[:, P:] = np.tril(np.ones((B, B), bool))
        for h in range(Hq):
            qt = torch.tensor(c["q"][r, :, h])[None, None]
            kt = torch.tensor(K[:, h // G])[None, None]
            vt = torch.tensor(V[:, h // G])[None, None]
            want = torch.nn.functional.scaled_dot_product_attention(
                qt, kt, vt, attn_mask=torch.tensor(mask)[None, None])[0, 0].numpy()
            np.testing.assert_allclose(out[r, :, h], want, atol=1e-12)
            z = c["q"][r, :, h] @ K[:, h // G].T / math.sqrt(D)
            z = np.where(mask, z, -np.inf)
            m = z.max(1)
            np.testing.assert_allclose(lse[r, :, h], m + np.log(np.exp(z - m[:, None]).sum(1)),
                                       atol=1e-12)


def test_softmax_online_reverse_tiles_agree():
    """A second algorithm: online (streaming max/sum) softmax over tiles taken
    in reverse order, written here in numpy."""
    c = _paged_case(lens=(7, 0, 19), seed=3)
    out, _ = oracle.block_softmax(c["q"], c["kb"], c["vb"], c["kp"], c["vp"], c["table"],
                                  c["lens"])
    R, B, Hq, D = c["q"].shape
    G = Hq // c["kb"].shape[2]
    for r in range(R):
        K = np.concatenate([c["dense_k"][r], c["kb"][r]], 0)
        V = np.concatenate([c["dense_v"][r], c["vb"][r]], 0)
        for h in range(Hq):
            for t in range(B):
                m, l, acc = -np.inf, 0.0, np.zeros(D)
                n = K.shape[0]
                for hi in range(n, 0, -3):
                    lo = max(hi - 3, 0)
                    z = K[lo:hi, h // G] @ c["q"][r, t, h] / math.sqrt(D)
                    m2 = max(m, z.max())
                    w = np.exp(z - m2)
                    acc = acc * math.exp(m - m2) + w @ V[lo:hi, h // G]
                    l = l * math.exp(m - m2) + w.sum()
                    m = m2
                np.testing.assert_allclose(out[r, t, h], acc / l, atol=1e-12)


def test_softmax_equal_keys_gives_mean_value():
    c = _paged_case(seed=5)
    c["kp"][:] = 0.5
    c["kb"][:] = 0.5
    out, _ = oracle.block_softmax(c["q"], c["kb"], c["vb"], c["kp"], c["vp"], c["table"],
                                  c["lens"])
    for r in range(3):
        for h in range(4):
            V = np.concatenate([c["dense_v"][r], c["vb"][r]], 0)[:, h // 2]
            np.testing.assert_allclose(out[r, :, h], np.broadcast_to(V.mean(0), (4, 16)),
                                       atol=1e-13)


def test_softmax_scale_zero_uniform_and_single_token():
    c = _paged_case(seed=6)
    out, lse = oracle.block_softmax(c["q"], c["kb"], c["vb"], c["kp"], c["vp"], c["table"],
                                    c["lens"], scale=0.0)
    for r in range(3):
        n = int(c["lens"][r]) + 4
        np.testing.assert_allclose(lse[r], math.log(n), atol=1e-13)
    # no prefix, one block token: the output is that token's value
    c = _paged_case(B=1, lens=(0, 0, 0), seed=7)
    out, _ = oracle.block_softmax(c["q"], c["kb"], c["vb"], c["kp"], c["vp"], c["table"],
                                  c["lens"])
    np.testing.assert_allclose(out[:, 0], c["vb"][:, 0][:, [0, 0, 1, 1]], atol=1e-15)


def test_softmax_causal_first_row_without_prefix():
    c = _paged_case(lens=(0, 0, 0), seed=8)
    out, _ = oracle.block_softmax(c["q"], c["kb"], c["vb"], c["kp"], c["vp"], c["table"],
                                  c["lens"], mask_mode=1)
    np.testing.assert_allclose(out[:, 0], c["vb"][:, 0][:, [0, 0, 1, 1]], atol=1e-15)


def test_gather_prefix_matches_scatter():
    c = _paged_case(lens=(9, 0, 16), p=4, seed=9)
    for r in range(3):
        got = oracle.gather_prefix(r, c["kp"], c["table"], c["lens"], 4)
        assert np.array_equal(got, c["dense_k"][r].reshape(got.shape))


def test_softmax_rejects_bad_page():
    c = _paged_case(seed=10)
    c["table"][2, 0] = c["kp"].shape[0]
    with pytest.raises(ValueError):
        oracle.block_softmax(c["q"], c["kb"], c["vb"], c["kp"], c["vp"], c["table"], c["lens"])


# ---------------------------------------------------------------- KV append


def test_append_then_gather_is_prefix_plus_block():
    """The state-update pass appends the block to the cache: gathering the
    longer prefix returns the old prefix followed by the appended tokens, and
    no other pool row changes."""
    c = _paged_case(R=3, B=4, lens=(5, 0, 12), p=4, seed=21, poison=True)
    # give every request room for the block: extra pages after its last one
    R, B, Hkv, D = c["kb"].shape
    num_pages = c["kp"].shape[0]
    extra = num_pages
    kp = np.concatenate([c["kp"], np.full((6,) + c["kp"].shape[1:], np.nan)], 0)
    vp = np.concatenate([c["vp"], np.full((6,) + c["vp"].shape[1:], np.nan)], 0)
    table = -np.ones((R, 8), np.int32)
    table[:, :c["table"].shape[1]] = c["table"]
    for r, P in enumerate(c["lens"]):
        first_free = -(-int(P) // 4)
        for q in range(first_free, -(-(int(P) + B) // 4)):
            table[r, q] = extra
            extra += 1
    append = np.array([4, 2, 0], np.int32)
    k2, v2 = oracle.append_kv(c["kb"], c["vb"], kp, vp, table, c["lens"], append)
    for r in range(R):
        P, n = int(c["lens"][r]), int(append[r])
        got = oracle.gather_prefix(r, k2, table, c["lens"] + append, 4)
        want = np.concatenate([c["dense_k"][r], c["kb"][r, :n]], 0)
        assert np.array_equal(got, want)
    # rows outside the appended positions are bit-identical (NaN included)
    touched = np.zeros(kp.shape[0] * 4, bool)
    for r in range(R):
        for t in range(int(append[r])):
            pos = int(c["lens"][r]) + t
            touched[table[r, pos // 4] * 4 + pos % 4] = True
    same = lambda a, b: np.array_equal(a.view(np.uint64), b.view(np.uint64))
    for pg in range(kp.shape[0]):
        for row in range(4):
            if not touched[pg * 4 + row]:
                assert same(k2[pg, :, row], kp[pg, :, row]) and same(v2[pg, :, row], vp[pg, :, row])


def test_append_rejects_overflow():
    c = _paged_case(R=3, B=4, lens=(5, 0, 12), p=4, seed=22)
    with pytest.raises(ValueError):
        oracle.append_kv(c["kb"], c["vb"], c["kp"], c["vp"], c["table"], c["lens"])
