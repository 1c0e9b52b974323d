"""Plain fp64 CPU oracle for FLARE's block-denoising attention step.

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The product library
never links or loads it, and it shares no code with the CUDA path.

The arithmetic lives in ``flare_oracle.c`` (fp64, optional OpenMP over
(request, head) items); this module compiles it with the system C compiler and
marshals numpy arrays into it.  What each routine computes, and which equation
of the paper it follows, is documented in the C file:

* :func:`gdr_per_token` -- gated delta rule token by token (Eq. per-step-fwd),
  block-end readout (Eq. noisy-block-fwd), commit at the accepted length.
* :func:`gdr_chunked` -- the same quantities through the chunkwise WY/UT form
  (Eq. chunk-state, Eq. f-blk); used only to pin :func:`gdr_per_token`.
* :func:`gdr_verify` -- the AR-Trust verify round: token-causal anchor/verify
  rows, bidirectional draft rows, and the states cached at each verify
  position (serving appendix, cache-and-scatter).
* :func:`verify_commit` -- the gather-scatter of the cached state at each
  request's accepted offset into every layer's state pool.
* :func:`two_stream_fwd` -- the noisy stream of the two-stream training
  forward (Eq. noisy-block-fwd): noisy blocks seeded with the clean state at
  their boundary, read at their block end.
* :func:`short_conv` -- the two-stream causal ShortConv of a block in its
  serving form (Eq. short-conv-noisy) and the commit of its W-1-token state.
* :func:`gather_prefix` -- dense copy of a request's paged prefix.
* :func:`block_softmax` -- softmax retrieval (Eq. softmax-retrieval) under the
  Diffusion-Trust block mask over the paged prefix plus the block.
* :func:`append_kv` -- the state-update pass's append of the block's keys and
  values to the paged cache.

Inputs may be bf16 (passed as raw ``uint16`` bit patterns), fp32 or fp64.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sysconfig
from pathlib import Path

import numpy as np

_HERE = Path(__file__).resolve().parent
_SRC = _HERE / "flare_oracle.c"
_LIB = _HERE / "_flare_oracle.so"
_lib = None

BF16, F32, F64 = 0, 1, 2


def build(force: bool = False) -> Path:
    """Compile the oracle into ``oracle/_flare_oracle.so`` (gcc, -O2, OpenMP if available)."""
    if _LIB.exists() and not force and _LIB.stat().st_mtime >= _SRC.stat().st_mtime:
        return _LIB
    cc = os.environ.get("CC", "gcc")
    tmp = _LIB.with_suffix(f".{os.getpid()}.tmp")
    base = [cc, "-O2", "-std=c11", "-shared", "-fPIC", str(_SRC), "-o", str(tmp), "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(str(_LIB))
        P, I, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
        lib.oracle_gdr_per_token.argtypes = [I] * 6 + [D, I, P, P, P, I, P, P, I, P, I, P, P, P, P, P, I]
        lib.oracle_gdr_per_token.restype = I
        lib.oracle_gdr_chunked.argtypes = [I] * 6 + [D, I, P, P, P, I, P, P, I, P, I, P, P, P, P, I]
        lib.oracle_gdr_chunked.restype = I
        lib.oracle_gather_prefix.argtypes = [I] * 7 + [P, P, P, P]
        lib.oracle_gather_prefix.restype = I
        lib.oracle_gdr_verify.argtypes = [I] * 6 + [D, I, I, P, P, P, I, P, P, I, P, I, P, P,
                                                    P, P, P, I]
        lib.oracle_gdr_verify.restype = I
        lib.oracle_block_softmax.argtypes = [I] * 8 + [D, I, I, P, P, P, P, P, P, P, P, P, P, I]
        lib.oracle_block_softmax.restype = I
        lib.oracle_two_stream_fwd.argtypes = [I] * 8 + [D, I, P, P, I, P, P, P, P, P, P, P, I, P,
                                                        P, P, P, I]
        lib.oracle_two_stream_fwd.restype = I
        lib.oracle_short_conv.argtypes = [I] * 6 + [P, P, I, P, I, P, P, P, P, P]
        lib.oracle_short_conv.restype = I
        lib.oracle_append_kv.argtypes = [I] * 8 + [P] * 7
        lib.oracle_append_kv.restype = I
        lib.oracle_max_threads.argtypes = []
        lib.oracle_max_threads.restype = I
        _lib = lib
    return _lib


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def _arr(x):
    """Return (contiguous numpy array, dtype code) for bf16/fp32/fp64 inputs.

    Accepts numpy arrays or CPU torch tensors; bf16 torch tensors are passed as
    their raw 16-bit patterns (the C side widens them exactly)."""
    if x is None:
        return None, F64
    if hasattr(x, "detach"):  # torch tensor
        import torch

        x = x.detach().cpu().contiguous()
        if x.dtype == torch.bfloat16:
            return x.view(torch.int16).numpy().view(np.uint16), BF16
        x = x.numpy()
    x = np.ascontiguousarray(x)
    if x.dtype == np.uint16:
        return x, BF16
    if x.dtype == np.float32:
        return x, F32
    if x.dtype == np.float64:
        return x, F64
    raise TypeError(f"unsupported oracle input dtype {x.dtype}")


def _i32(x):
    if hasattr(x, "detach"):
        x = x.detach().cpu().numpy()
    return np.ascontiguousarray(np.asarray(x, dtype=np.int32))


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _gdr_args(q, k, v, log_decay, beta, state_pool, state_slot, accept_len):
    qa, qdt = _arr(q)
    ka, kdt = _arr(k)
    va, vdt = _arr(v)
    if q is not None and qdt != kdt:
        raise TypeError("q and k must share an element type")
    if kdt != vdt:
        raise TypeError("k and v must share an element type")
    ga, gdt = _arr(log_decay)
    ba, bdt = _arr(beta)
    if gdt != bdt:
        raise TypeError("log_decay and beta must share an element type")
    sa, sdt = _arr(state_pool)
    slot = _i32(state_slot)
    acc = None if accept_len is None else _i32(accept_len)
    R, B, Hk, dk = ka.shape
    Hv, dv = va.shape[2], va.shape[3]
    return dict(qa=qa, ka=ka, va=va, ga=ga, ba=ba, sa=sa, slot=slot, acc=acc, dt=kdt, gdt=gdt,
                sdt=sdt, R=R, B=B, Hk=Hk, Hv=Hv, dk=dk, dv=dv, nslots=sa.shape[0])


def gdr_per_token(q, k, v, log_decay, beta, state_pool, state_slot, accept_len=None, *,
                  scale=None, blockend=True, causal=False, state=True, nthreads=0):
    """Gated delta rule over one block, token by token (Eq. per-step-fwd).

    Shapes: q, k [R,B,Hk,dk]; v [R,B,Hv,dv]; log_decay, beta [R,B,Hv];
    state_pool [slots,Hv,dk,dv]; state_slot [R]; accept_len [R] or None (= B).
    Returns a dict with fp64 arrays ``blockend`` [R,B,Hv,dv] (s S_B^T q_l),
    ``causal`` [R,B,Hv,dv] (s S_t^T q_t) and ``state`` [R,Hv,dk,dv]
    (S at the accepted length), each present when asked for.
    """
    a = _gdr_args(q, k, v, log_decay, beta, state_pool, state_slot, accept_len)
    R, B, Hv, dk, dv = a["R"], a["B"], a["Hv"], a["dk"], a["dv"]
    s = 1.0 / np.sqrt(dk) if scale is None else float(scale)
    ob = np.zeros((R, B, Hv, dv)) if blockend else None
    oc = np.zeros((R, B, Hv, dv)) if causal else None
    st = np.zeros((R, Hv, dk, dv)) if state else None
    if (blockend or causal) and q is None:
        raise ValueError("q is required for a readout")
    rc = _load().oracle_gdr_per_token(
        R, B, a["Hk"], Hv, dk, dv, s, a["dt"], _ptr(a["qa"]), _ptr(a["ka"]), _ptr(a["va"]),
        a["gdt"], _ptr(a["ga"]), _ptr(a["ba"]), a["sdt"], _ptr(a["sa"]), a["nslots"],
        _ptr(a["slot"]), _ptr(a["acc"]), _ptr(ob), _ptr(oc), _ptr(st), int(nthreads))
    if rc != 0:
        raise ValueError("oracle_gdr_per_token: invalid state slot or accepted length")
    return {k_: v_ for k_, v_ in (("blockend", ob), ("causal", oc), ("state", st)) if v_ is not None}


def gdr_chunked(q, k, v, log_decay, beta, state_pool, state_slot, accept_len=None, *,
                scale=None, nthreads=0):
    """Chunkwise WY/UT form of the same block (Eq. chunk-state, Eq. f-blk).

    Returns ``blockend`` and ``state`` like :func:`gdr_per_token`."""
    if q is None:
        raise ValueError("gdr_chunked forms the block-end readout and needs q")
    a = _gdr_args(q, k, v, log_decay, beta, state_pool, state_slot, accept_len)
    R, B, Hv, dk, dv = a["R"], a["B"], a["Hv"], a["dk"], a["dv"]
    s = 1.0 / np.sqrt(dk) if scale is None else float(scale)
    ob = np.zeros((R, B, Hv, dv))
    st = np.zeros((R, Hv, dk, dv))
    rc = _load().oracle_gdr_chunked(
        R, B, a["Hk"], Hv, dk, dv, s, a["dt"], _ptr(a["qa"]), _ptr(a["ka"]), _ptr(a["va"]),
        a["gdt"], _ptr(a["ga"]), _ptr(a["ba"]), a["sdt"], _ptr(a["sa"]), a["nslots"],
        _ptr(a["slot"]), _ptr(a["acc"]), _ptr(ob), _ptr(st), int(nthreads))
    if rc != 0:
        raise ValueError("oracle_gdr_chunked: invalid state slot or accepted length")
    return {"blockend": ob, "state": st}


def gdr_verify(q, k, v, log_decay, beta, state_pool, state_slot, verify_len, max_verify, *,
               scale=None, nthreads=0):
    """AR-Trust verify round of one gated-delta-rule layer.

    Shapes: q, k [R,L,Hk,dk]; v [R,L,Hv,dv]; log_decay, beta [R,L,Hv];
    state_pool [slots,Hv,dk,dv]; state_slot, verify_len [R] (K_r, the number
    of held drafts being verified, 0..min(max_verify, L-1)).
    Returns fp64 ``out`` [R,L,Hv,dv] (rows t <= K_r: s S_{t+1}^T q_t; later
    rows: s S_L^T q_t), ``records`` [R,max_verify,Hv,dk,dv] (record t < K_r is
    S_{t+1}, the state after the anchor and t drafts; the rest stay zero) and
    ``state`` [R,Hv,dk,dv] (S_{K_r+1}, the live state after every verify
    token)."""
    a = _gdr_args(q, k, v, log_decay, beta, state_pool, state_slot, None)
    R, L, Hv, dk, dv = a["R"], a["B"], a["Hv"], a["dk"], a["dv"]
    s = 1.0 / np.sqrt(dk) if scale is None else float(scale)
    vl = _i32(verify_len)
    out = np.zeros((R, L, Hv, dv))
    rec = np.zeros((R, max_verify, Hv, dk, dv))
    st = np.zeros((R, Hv, dk, dv))
    rc = _load().oracle_gdr_verify(
        R, L, a["Hk"], Hv, dk, dv, s, int(max_verify), a["dt"], _ptr(a["qa"]), _ptr(a["ka"]),
        _ptr(a["va"]), a["gdt"], _ptr(a["ga"]), _ptr(a["ba"]), a["sdt"], _ptr(a["sa"]),
        a["nslots"], _ptr(a["slot"]), _ptr(vl), _ptr(out), _ptr(rec), _ptr(st), int(nthreads))
    if rc != 0:
        raise ValueError("oracle_gdr_verify: invalid state slot or verify length")
    return {"out": out, "records": rec, "state": st}


def verify_commit(records, pools, state_slot, accept, verify_len):
    """Gather-scatter commit of a verify round (serving appendix, path (b)).

    records: per layer [R, max_verify, Hv, dk, dv]; pools: per layer
    [slots, Hv, dk, dv]; accept[r] in [0, verify_len[r]] is the number of
    accepted drafts.  Returns copies of the pools where, for every layer and
    every request with accept[r] < verify_len[r], slot state_slot[r] holds
    records[r][accept[r]] bit for bit; a request that accepted every draft
    already has S^(K) in the pool and is left alone.  Raises ValueError on an
    out-of-range slot, accepted offset or verify length."""
    slot, acc, vl = _i32(state_slot), _i32(accept), _i32(verify_len)
    outs = [np.array(p, copy=True) for p in pools]
    for rec, pool in zip(records, outs):
        R, max_verify = rec.shape[0], rec.shape[1]
        for r in range(R):
            if not (0 <= slot[r] < pool.shape[0] and 0 <= vl[r] <= max_verify
                    and 0 <= acc[r] <= vl[r]):
                raise ValueError("verify_commit: invalid slot, accepted offset or verify length")
            if acc[r] < vl[r]:
                pool[slot[r]] = rec[r, acc[r]]
    return outs


def two_stream_fwd(clean, noisy, S_init, block_len, chunk_len, *, chunk_states=None,
                   record_chunk_states=False, scale=None, nthreads=0):
    """Noisy stream of the two-stream GDR training forward (Eq. noisy-block-fwd).

    clean = (k [N,L,Hk,dk], v [N,L,Hv,dv], g [N,L,Hv], beta [N,L,Hv]);
    noisy = (q, k, v, g, beta) with the same shapes (q like k); S_init
    [N,Hv,dk,dv] is the clean state before position 0.  With chunk_states
    [N,Hv,L/C,dk,dv] the clean state is reset to them at every chunk start.
    Returns fp64 ``out`` [N,L,Hv,dv] and, when asked, ``chunk_states`` (the
    clean state at each chunk start)."""
    k, v, g, beta = clean
    qn, kn, vn, gn, bn = noisy
    ka, kdt = _arr(k)
    va, vdt = _arr(v)
    qna, qdt = _arr(qn)
    kna, kndt = _arr(kn)
    vna, vndt = _arr(vn)
    if len({kdt, vdt, qdt, kndt, vndt}) != 1:
        raise TypeError("activations must share an element type")
    ga, gdt = _arr(g)
    ba, bdt = _arr(beta)
    gna, gndt = _arr(gn)
    bna, bndt = _arr(bn)
    if len({gdt, bdt, gndt, bndt}) != 1:
        raise TypeError("gates must share an element type")
    sa, sdt = _arr(S_init)
    ci = None
    if chunk_states is not None:
        ci, cdt = _arr(chunk_states)
        if cdt != sdt:
            raise TypeError("chunk states and S_init must share an element type")
    N, L, Hk, dk = ka.shape
    Hv, dv = va.shape[2], va.shape[3]
    s = 1.0 / np.sqrt(dk) if scale is None else float(scale)
    out = np.zeros((N, L, Hv, dv))
    co = np.zeros((N, Hv, L // chunk_len, dk, dv)) if record_chunk_states else None
    rc = _load().oracle_two_stream_fwd(
        N, L, Hk, Hv, dk, dv, int(block_len), int(chunk_len), s, kdt, _ptr(ka), _ptr(va), gdt,
        _ptr(ga), _ptr(ba), _ptr(qna), _ptr(kna), _ptr(vna), _ptr(gna), _ptr(bna), sdt, _ptr(sa),
        _ptr(ci), _ptr(out), _ptr(co), int(nthreads))
    if rc != 0:
        raise ValueError("oracle_two_stream_fwd: block length must divide the chunk length, "
                         "and the chunk length the sequence length")
    res = {"out": out}
    if co is not None:
        res["chunk_states"] = co
    return res


def short_conv(x, conv_state, state_slot, weight, bias=None, *, silu=True, accept_len=None):
    """Two-stream causal ShortConv of a block, serving form (Eq. short-conv-noisy).

    Shapes: x [R,B,C]; conv_state [slots, W-1, C] (the last W-1 clean tokens
    before each request's block, oldest first); state_slot [R]; weight [C,W]
    (weight[c, i] multiplies lag i); bias [C] or None; accept_len [R] or None.
    Returns fp64 ``out`` [R,B,C] and, when accept_len is given, ``state``
    [R, W-1, C], the last W-1 rows of (old state ++ the first accept_len[r]
    block rows)."""
    xa, xdt = _arr(x)
    sa, sdt = _arr(conv_state)
    if sdt != xdt:
        raise TypeError("x and conv_state must share an element type")
    wa, wdt = _arr(weight)
    ba = None
    if bias is not None:
        ba, bdt = _arr(bias)
        if bdt != wdt:
            raise TypeError("weight and bias must share an element type")
    slot = _i32(state_slot)
    acc = None if accept_len is None else _i32(accept_len)
    R, B, C = xa.shape
    W = wa.shape[1]
    out = np.zeros((R, B, C))
    st = np.zeros((R, W - 1, C)) if acc is not None else None
    rc = _load().oracle_short_conv(R, B, C, W, int(bool(silu)), xdt, _ptr(xa), _ptr(sa),
                                   sa.shape[0], _ptr(slot), wdt, _ptr(wa), _ptr(ba), _ptr(acc),
                                   _ptr(out), _ptr(st))
    if rc != 0:
        raise ValueError("oracle_short_conv: invalid slot, width or accepted length")
    res = {"out": out}
    if st is not None:
        res["state"] = st
    return res


def gather_prefix(r, pool, page_table, prefix_len, page_size):
    """Dense fp64 copy [P_r, Hkv, D] of request r's paged prefix from one pool."""
    pa, pdt = _arr(pool)
    tab = _i32(page_table)
    lens = _i32(prefix_len)
    num_pages, Hkv, p, D = pa.shape
    assert p == page_size
    out = np.zeros((int(lens[r]), Hkv, D))
    rc = _load().oracle_gather_prefix(int(r), Hkv, D, page_size, num_pages, tab.shape[1], pdt,
                                      _ptr(pa), _ptr(tab), _ptr(lens), _ptr(out))
    if rc != 0:
        raise ValueError("oracle_gather_prefix: invalid page id or prefix length")
    return out


def block_softmax(q, k_blk, v_blk, k_pool, v_pool, page_table, prefix_len, *, scale=None,
                  mask_mode=0, row_type=None, nthreads=0):
    """Block-query softmax attention over paged prefix + block (Eq. softmax-retrieval).

    mask_mode 0: every block row sees every block token (denoise pass);
    mask_mode 1: block row t sees block tokens 0..t (state-update pass);
    mask_mode 2 / 3: per-row types, ``row_type`` uint8 [B] (shared) or [R,B]
    (per request); type 0 rows are token-causal, type 1 rows bidirectional.
    Returns (out [R,B,Hq,D], lse [R,B,Hq]) in fp64."""
    qa, dt = _arr(q)
    kb, _ = _arr(k_blk)
    vb, _ = _arr(v_blk)
    kp, _ = _arr(k_pool)
    vp, _ = _arr(v_pool)
    tab = _i32(page_table)
    lens = _i32(prefix_len)
    R, B, Hq, D = qa.shape
    Hkv = kb.shape[2]
    num_pages, _, p, _ = kp.shape
    sc = 1.0 / np.sqrt(D) if scale is None else float(scale)
    out = np.zeros((R, B, Hq, D))
    lse = np.zeros((R, B, Hq))
    rt = None
    if mask_mode in (2, 3):
        if hasattr(row_type, "detach"):
            row_type = row_type.detach().cpu().numpy()
        rt = np.ascontiguousarray(np.asarray(row_type, dtype=np.uint8))
        if rt.shape != ((B,) if mask_mode == 2 else (R, B)):
            raise ValueError("row_type shape does not match the mask mode")
    rc = _load().oracle_block_softmax(
        R, B, Hq, Hkv, D, p, num_pages, tab.shape[1], sc, int(mask_mode), dt, _ptr(qa), _ptr(kb),
        _ptr(vb), _ptr(kp), _ptr(vp), _ptr(tab), _ptr(lens), _ptr(rt), _ptr(out), _ptr(lse),
        int(nthreads))
    if rc != 0:
        raise ValueError("oracle_block_softmax: invalid page id, prefix length or row type")
    return out, lse


def append_kv(k_blk, v_blk, k_pool, v_pool, page_table, prefix_len, append_len=None):
    """Returns copies of (k_pool, v_pool) with the first append_len[r] (default B)
    block tokens of every request written at prefix positions prefix_len[r] + t.
    Works on any element type bit for bit (numpy arrays or CPU torch tensors)."""
    def raw(x):
        if hasattr(x, "detach"):
            import torch

            x = x.detach().cpu().contiguous()
            if x.dtype == torch.bfloat16:
                return x.view(torch.int16).numpy().view(np.uint16)
            return x.numpy()
        return np.ascontiguousarray(x)
    kb, vb = raw(k_blk), raw(v_blk)
    kp, vp = raw(k_pool).copy(), raw(v_pool).copy()
    tab, lens = _i32(page_table), _i32(prefix_len)
    acc = None if append_len is None else _i32(append_len)
    R, B, Hkv, D = kb.shape
    num_pages, _, p, _ = kp.shape
    rc = _load().oracle_append_kv(R, B, Hkv, D, p, num_pages, tab.shape[1], kb.itemsize,
                                  _ptr(kb), _ptr(vb), _ptr(kp), _ptr(vp), _ptr(tab), _ptr(lens),
                                  _ptr(acc))
    if rc != 0:
        raise ValueError("oracle_append_kv: invalid page id or length")
    return kp, vp
