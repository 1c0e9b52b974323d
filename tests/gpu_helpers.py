"""Shared plumbing of the GPU parity tests: run the C-ABI calls on a workload
and produce the oracle's answer for the same inputs."""
from __future__ import annotations

import math

import numpy as np
import torch

import oracle
from paper_2606_01774_gb300 import flare, workloads

# Tolerances (the accuracy the serving path must keep: max-abs 2e-2 on bf16
# outputs, relative Frobenius 1e-3 on fp32 committed states).  The tighter
# relative bounds on outputs follow from the
# arithmetic: bf16 output rounding is 2^-9 relative, bf16 tensor-core operands
# add a few 2^-9 more; fp32 paths carry ~1e-6.
OUT_MAX_ABS = 2e-2
OUT_REL_FRO = {"bf16": 1e-2, "f32": 1e-4}
STATE_REL_FRO = 1e-3


def act_code(spec):
    return flare.FLARE_DT_BF16 if spec.act_dtype == "bf16" else flare.FLARE_DT_F32


def linear_desc(spec, nslots):
    return flare.linear_desc(spec.num_requests, spec.block_len, spec.num_qk_heads,
                             spec.num_v_heads, spec.head_dim_k, spec.head_dim_v, nslots,
                             act_code(spec), 1.0 / math.sqrt(spec.head_dim_k))


def softmax_desc(spec, w, mode=flare.FLARE_MASK_BLOCK_BIDIR, row_type=None):
    return flare.softmax_desc(spec.num_requests, spec.block_len, spec.num_q_heads,
                              spec.num_kv_heads, spec.head_dim, spec.page_size,
                              w.k_pool.shape[0], w.page_table.shape[1], act_code(spec),
                              1.0 / math.sqrt(spec.head_dim), mode, row_type)


def oracle_states(w, requests=None):
    """fp64 S0 [len(requests), Hv, dk, dv]: the oracle's gated delta rule over each
    request's random prefix tokens, starting from the zero state."""
    spec = w.spec
    req = list(range(spec.num_requests)) if requests is None else list(requests)
    sp = w.state_prefix
    idx = torch.tensor(req, device=sp.k.device)
    zero = np.zeros((1, spec.num_v_heads, spec.head_dim_k, spec.head_dim_v), np.float32)
    o = oracle.gdr_per_token(None, sp.k[idx].cpu(), sp.v[idx].cpu(), sp.log_decay[idx].cpu(),
                             sp.beta[idx].cpu(), zero, np.zeros(len(req), np.int32), None,
                             blockend=False)
    return o["state"]


def install_states(w, requests=None, fill_rest=True):
    """Write oracle-built S0 (rounded to fp32) into the pool slots of `requests`;
    other used slots get a seeded random state of similar scale (their outputs
    are not compared)."""
    spec = w.spec
    req = list(range(spec.num_requests)) if requests is None else list(requests)
    S0 = torch.from_numpy(oracle_states(w, req)).float().to(w.state_pool.device)
    slots = w.state_slot.long()
    if fill_rest and len(req) < spec.num_requests:
        g = torch.Generator(device=w.state_pool.device)
        g.manual_seed(1000 + spec.seed)
        rest = torch.randn(spec.num_requests, spec.num_v_heads, spec.head_dim_k,
                           spec.head_dim_v, generator=g, device=w.state_pool.device) * 0.05
        w.state_pool[slots] = rest
    w.state_pool[slots[torch.tensor(req, device=slots.device)]] = S0
    return S0


def status_word(device):
    return torch.zeros(1, dtype=torch.int32, device=device)


def run_linear(w, step=0):
    spec = w.spec
    blk = w.denoise[step]
    out = torch.empty_like(blk.v)
    st = status_word(blk.v.device)
    rc = flare.flare_block_linear_attn(linear_desc(spec, w.state_pool.shape[0]), blk.q, blk.k,
                                       blk.v, blk.log_decay, blk.beta, w.state_pool, w.state_slot,
                                       out, st)
    flare.check(rc, "flare_block_linear_attn")
    rc, bits = flare.flare_read_status(st)
    assert bits == 0 and rc == flare.FLARE_OK, bits
    return out


def run_commit(w, pool, causal=False, accept_len=None):
    spec = w.spec
    blk = w.commit
    acc = w.accept_len if accept_len is None else accept_len
    co = torch.empty_like(blk.v) if causal else None
    st = status_word(blk.v.device)
    rc = flare.flare_commit_state(linear_desc(spec, pool.shape[0]), blk.q, blk.k, blk.v,
                                  blk.log_decay, blk.beta, pool, w.state_slot, acc, co, st)
    flare.check(rc, "flare_commit_state")
    rc, bits = flare.flare_read_status(st)
    assert bits == 0 and rc == flare.FLARE_OK, bits
    return co


def run_softmax(w, step=0, mode=flare.FLARE_MASK_BLOCK_BIDIR, want_lse=True, row_type=None):
    spec = w.spec
    sb = w.softmax[step]
    desc = softmax_desc(spec, w, mode, row_type)
    ws_bytes = flare.flare_softmax_workspace_size(desc)
    ws = torch.empty(max(ws_bytes, 1), dtype=torch.uint8, device=sb.q.device)
    out = torch.empty_like(sb.q)
    lse = torch.empty(sb.q.shape[:3], dtype=torch.float32, device=sb.q.device) if want_lse else None
    st = status_word(sb.q.device)
    rc = flare.flare_block_softmax_attn(desc, sb.q, sb.k_blk, sb.v_blk, w.k_pool, w.v_pool,
                                        w.page_table, w.prefix_len, out, lse, ws, ws_bytes, st)
    flare.check(rc, "flare_block_softmax_attn")
    rc, bits = flare.flare_read_status(st)
    assert bits == 0 and rc == flare.FLARE_OK, bits
    return out, lse


def oracle_linear(w, step=0, requests=None):
    spec = w.spec
    req = list(range(spec.num_requests)) if requests is None else list(requests)
    blk = w.denoise[step]
    i = torch.tensor(req, device=blk.q.device)
    slots = w.state_slot[i].cpu()
    pool = w.state_pool[slots.long()].cpu()
    o = oracle.gdr_per_token(blk.q[i].cpu(), blk.k[i].cpu(), blk.v[i].cpu(),
                             blk.log_decay[i].cpu(), blk.beta[i].cpu(), pool,
                             np.arange(len(req), dtype=np.int32), None,
                             scale=1.0 / math.sqrt(spec.head_dim_k), state=False)
    return o["blockend"]


def oracle_commit(w, pool_before, requests=None, causal=False, accept_len=None):
    spec = w.spec
    req = list(range(spec.num_requests)) if requests is None else list(requests)
    blk = w.commit
    acc = (w.accept_len if accept_len is None else accept_len)
    i = torch.tensor(req, device=blk.k.device)
    slots = w.state_slot[i].cpu()
    pool = pool_before[slots.long()].cpu()
    o = oracle.gdr_per_token(blk.q[i].cpu(), blk.k[i].cpu(), blk.v[i].cpu(),
                             blk.log_decay[i].cpu(), blk.beta[i].cpu(), pool,
                             np.arange(len(req), dtype=np.int32), acc[i].cpu(),
                             scale=1.0 / math.sqrt(spec.head_dim_k), blockend=False,
                             causal=causal)
    return o


def oracle_softmax(w, step=0, requests=None, mode=0, row_type=None):
    """row_type: [B] (mode 2) or [R,B] (mode 3, rows of `requests` taken here)."""
    spec = w.spec
    req = list(range(spec.num_requests)) if requests is None else list(requests)
    sb = w.softmax[step]
    i = torch.tensor(req, device=sb.q.device)
    rt = None
    if mode == 2:
        rt = row_type.cpu()
    elif mode == 3:
        rt = row_type[i].cpu()
    return oracle.block_softmax(sb.q[i].cpu(), sb.k_blk[i].cpu(), sb.v_blk[i].cpu(),
                                w.k_pool.cpu(), w.v_pool.cpu(), w.page_table[i].cpu(),
                                w.prefix_len[i].cpu(), scale=1.0 / math.sqrt(spec.head_dim),
                                mask_mode=mode, row_type=rt)


def run_verify_linear(w, max_verify, verify_len=None, records=None, expect_bits=0):
    """AR-Trust verify round of the linear layer on w.denoise[0] (updates
    w.state_pool in place).  Returns (out, records)."""
    spec = w.spec
    blk = w.denoise[0]
    vl = w.verify_len if verify_len is None else verify_len
    out = torch.empty_like(blk.v)
    if records is None:
        records = torch.full((spec.num_requests, max_verify, spec.num_v_heads, spec.head_dim_k,
                              spec.head_dim_v), float("nan"), device=blk.v.device)
    st = status_word(blk.v.device)
    rc = flare.flare_verify_linear_attn(linear_desc(spec, w.state_pool.shape[0]), max_verify,
                                        blk.q, blk.k, blk.v, blk.log_decay, blk.beta,
                                        w.state_pool, w.state_slot, vl, out,
                                        records if max_verify else None, st)
    flare.check(rc, "flare_verify_linear_attn")
    rc, bits = flare.flare_read_status(st)
    assert bits == expect_bits, bits
    return out, records


def oracle_verify(w, pool_before, max_verify, requests=None, verify_len=None):
    spec = w.spec
    req = list(range(spec.num_requests)) if requests is None else list(requests)
    blk = w.denoise[0]
    vl = w.verify_len if verify_len is None else verify_len
    i = torch.tensor(req, device=blk.k.device)
    slots = w.state_slot[i].cpu()
    pool = pool_before[slots.long()].cpu()
    return oracle.gdr_verify(blk.q[i].cpu(), blk.k[i].cpu(), blk.v[i].cpu(),
                             blk.log_decay[i].cpu(), blk.beta[i].cpu(), pool,
                             np.arange(len(req), dtype=np.int32), vl[i].cpu(), max_verify,
                             scale=1.0 / math.sqrt(spec.head_dim_k))


def rel_fro(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def assert_out_close(gpu, ref, act_dtype, what=""):
    g = gpu.detach().double().cpu().numpy() if hasattr(gpu, "detach") else np.asarray(gpu)
    assert np.isfinite(g).all(), f"{what}: non-finite GPU output"
    err = np.abs(g - ref).max()
    rf = rel_fro(g, ref)
    assert err <= OUT_MAX_ABS, f"{what}: max-abs {err:.3e} > {OUT_MAX_ABS}"
    assert rf <= OUT_REL_FRO[act_dtype], f"{what}: rel-Frobenius {rf:.3e}"
    return err, rf


def assert_states_close(gpu, ref, what=""):
    """Relative Frobenius error per (request, head) state."""
    g = gpu.detach().double().cpu().numpy() if hasattr(gpu, "detach") else np.asarray(gpu)
    assert np.isfinite(g).all(), f"{what}: non-finite state"
    worst = 0.0
    for idx in np.ndindex(*g.shape[:2]):
        worst = max(worst, rel_fro(g[idx], ref[idx]))
    assert worst <= STATE_REL_FRO, f"{what}: state rel-Frobenius {worst:.3e}"
    return worst


def reduced(spec, num_requests=3, prefix_lo=None, prefix_hi=None):
    """Same layer shapes with fewer requests and (optionally) shorter prefixes:
    sizes the oracle finishes in seconds that still span several tiles."""
    kw = dict(num_requests=num_requests)
    if prefix_lo is not None:
        kw.update(prefix_lo=prefix_lo, prefix_hi=prefix_hi)
    return spec.replace(**kw)


def gen(spec, device="cuda"):
    return workloads.generate(spec, device)
