"""Pins for the two-stream training-forward part of the CPU oracle (noisy
stream of the GDR, Eq. noisy-block-fwd; what Route II computes).

Checked against: the Diffusion-Trust denoise readout (one noisy block over the
whole sequence is the serving denoise pass), the independent chunkwise WY form
for the clean chunk states (Eq. chunk-state / f-blk), the case of identical
clean and noisy streams (each noisy block then ends in the clean state), the
beta = 0 closed form, and the paper's statement that noisy blocks are mutually
independent.
"""
import numpy as np
import pytest

import oracle


def _unit(x):
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


def _stream(g, N, L, Hk, Hv, dk, dv, q=True):
    k = _unit(g.standard_normal((N, L, Hk, dk)))
    v = g.standard_normal((N, L, Hv, dv))
    gg = -np.log1p(np.exp(g.standard_normal((N, L, Hv))))
    b = 1.0 / (1.0 + np.exp(-g.standard_normal((N, L, Hv))))
    if q:
        return _unit(g.standard_normal((N, L, Hk, dk))), k, v, gg, b
    return k, v, gg, b


def _case(N=2, L=24, Hk=2, Hv=4, dk=8, dv=6, seed=0):
    g = np.random.default_rng(seed)
    clean = _stream(g, N, L, Hk, Hv, dk, dv, q=False)
    noisy = _stream(g, N, L, Hk, Hv, dk, dv)
    S0 = g.standard_normal((N, Hv, dk, dv)) * 0.3
    return clean, noisy, S0


def test_one_block_is_the_denoise_readout():
    """B = C = L: the single noisy block starts from S_init, which is the
    serving denoise pass (block-end readout from the committed state)."""
    clean, noisy, S0 = _case(L=12)
    N, L = S0.shape[0], 12
    o = oracle.two_stream_fwd(clean, noisy, S0, L, L)["out"]
    q, k, v, g, b = noisy
    want = oracle.gdr_per_token(q, k, v, g, b, S0, np.arange(N, dtype=np.int32), state=False)
    np.testing.assert_allclose(o, want["blockend"], rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("B,C", [(1, 4), (4, 8), (3, 12)])
def test_chunk_states_match_the_chunkwise_form(B, C):
    """The recorded clean state at chunk c is f_blk applied to S_init over the
    first c C clean tokens: the independent chunkwise WY implementation."""
    clean, noisy, S0 = _case(L=24, seed=B + C)
    N = S0.shape[0]
    res = oracle.two_stream_fwd(clean, noisy, S0, B, C, record_chunk_states=True)
    k, v, g, b = clean
    for c in range(24 // C):
        acc = np.full(N, c * C, np.int32)
        want = oracle.gdr_chunked(noisy[0], k, v, g, b, S0, np.arange(N, dtype=np.int32),
                                  acc)["state"]
        np.testing.assert_allclose(res["chunk_states"][:, :, c], want, rtol=1e-10, atol=1e-12)


def test_identical_streams_read_the_clean_state():
    """With the noisy stream equal to the clean one each noisy block ends in
    the clean state at the block end, so block b's rows read S_{(b+1)B}."""
    clean, noisy, S0 = _case(L=16, seed=5)
    k, v, g, b = clean
    q = noisy[0]
    N, B = S0.shape[0], 4
    o = oracle.two_stream_fwd(clean, (q, k, v, g, b), S0, B, 8)["out"]
    for blk in range(16 // B):
        n_tok = (blk + 1) * B
        want = oracle.gdr_per_token(q[:, :n_tok], k[:, :n_tok], v[:, :n_tok], g[:, :n_tok],
                                    b[:, :n_tok], S0, np.arange(N, dtype=np.int32),
                                    state=False)["blockend"]
        np.testing.assert_allclose(o[:, blk * B:n_tok], want[:, blk * B:], rtol=1e-12,
                                   atol=1e-12)


def test_noisy_beta_zero_closed_form():
    """beta~ = 0: the noisy block only decays its seed, out_l =
    s exp(sum of the block's noisy log-gates) S_{bB}^T q~_l."""
    clean, noisy, S0 = _case(L=12, seed=7)
    q, k, v, g, b = noisy
    noisy = (q, k, v, g, np.zeros_like(b))
    B = 3
    res = oracle.two_stream_fwd(clean, noisy, S0, B, B, record_chunk_states=True)
    N, L, Hv = g.shape
    Hk, dk = q.shape[2], q.shape[3]
    for blk in range(L // B):
        Sb = res["chunk_states"][:, :, blk]  # C = B: every block start is a chunk start
        G = np.exp(g[:, blk * B:(blk + 1) * B].sum(1))  # [N, Hv]
        for n in range(N):
            for j in range(Hv):
                for l in range(blk * B, (blk + 1) * B):
                    want = G[n, j] * Sb[n, j].T @ q[n, l, j * Hk // Hv] / np.sqrt(dk)
                    np.testing.assert_allclose(res["out"][n, l, j], want, rtol=1e-12,
                                               atol=1e-14)


def test_noisy_blocks_are_independent():
    """Changing the noisy tokens of one block changes that block's outputs
    only; changing a clean token changes only the blocks after it."""
    clean, noisy, S0 = _case(L=16, seed=9)
    B, C = 4, 8
    base = oracle.two_stream_fwd(clean, noisy, S0, B, C)["out"]
    q, k, v, g, b = (x.copy() for x in noisy)
    v[:, 5] += 1.0  # noisy token in block 1
    o = oracle.two_stream_fwd(clean, (q, k, v, g, b), S0, B, C)["out"]
    changed = np.abs(o - base).max(axis=(0, 2, 3)) > 0
    assert changed.tolist() == [t // B == 1 for t in range(16)]
    kc, vc, gc, bc = (x.copy() for x in clean)
    vc[:, 9] += 1.0  # clean token in block 2
    o = oracle.two_stream_fwd((kc, vc, gc, bc), noisy, S0, B, C)["out"]
    changed = np.abs(o - base).max(axis=(0, 2, 3)) > 0
    assert changed.tolist() == [t // B >= 3 for t in range(16)]


def test_given_chunk_states_restart_each_chunk():
    """Chunk states passed in replace the propagated clean state at each
    chunk start: the recorded ones reproduce the outputs, and a changed one
    changes only its own chunk."""
    clean, noisy, S0 = _case(L=16, seed=11)
    B, C = 2, 8
    res = oracle.two_stream_fwd(clean, noisy, S0, B, C, record_chunk_states=True)
    cs = res["chunk_states"]
    again = oracle.two_stream_fwd(clean, noisy, S0, B, C, chunk_states=cs)["out"]
    np.testing.assert_allclose(again, res["out"], rtol=1e-13, atol=1e-14)
    cs2 = cs.copy()
    cs2[:, :, 0] *= 2.0
    o = oracle.two_stream_fwd(clean, noisy, S0, B, C, chunk_states=cs2)["out"]
    changed = np.abs(o - res["out"]).max(axis=(0, 2, 3)) > 0
    assert changed.tolist() == [t < C for t in range(16)]


def test_bad_lengths_rejected():
    clean, noisy, S0 = _case(L=12)
    with pytest.raises(ValueError):
        oracle.two_stream_fwd(clean, noisy, S0, 5, 10)
    with pytest.raises(ValueError):
        oracle.two_stream_fwd(clean, noisy, S0, 4, 8)
