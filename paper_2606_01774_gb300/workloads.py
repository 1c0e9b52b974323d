"""Seeded synthetic workloads shaped like FLARE's serving batches.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic, so both the CUDA path and the CPU oracle can take their
inputs from it.  The recurrent state S0 that a request carries into a block is
NOT built here: the generator returns the random prefix tokens, and each caller
runs the gated delta rule over them with its own implementation.

Value distributions (the serving workloads of the paper, synthetic):
  * linear layer: q, k ~ N(0,1) then L2-normalised per head; v ~ N(0,1);
    log-gate g = -softplus(N(0,1)) (so the gate exp(g) = exp(-softplus(x)));
    beta = sigmoid(N(0,1)).
  * softmax layer: q, k, v ~ N(0,1).
  * prefix lengths ~ U{lo..hi}; the paged pool holds each request's pages at
    a random permutation of page ids, plus >= 5 % spare pages.  Spare pages,
    unused page-table entries (-1), the rows past the prefix end in a request's
    last page, and unused state slots are poisoned with NaN so that a stray
    read shows up in the outputs.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch


@dataclass(frozen=True)
class WorkloadSpec:
    name: str
    description: str
    num_requests: int
    block_len: int
    num_qk_heads: int
    num_v_heads: int
    head_dim_k: int
    head_dim_v: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    page_size: int
    prefix_lo: int
    prefix_hi: int
    act_dtype: str  # "bf16" or "f32"
    denoise_steps: int
    accept: str  # "full", "fixed" or "uniform"
    accept_fixed: int
    state_prefix_tokens: int
    seed: int
    spare_slots: int = 4
    # AR-Trust verify round: speculation horizon N (0 = not a verify workload).
    # The block is [anchor, d_0 .. d_{K-1}, MASK ...] of length block_len
    # (2N - 1 at steady state); K ~ U{0..N-1} held drafts per request (0 is a
    # cold start) and the accepted offset a ~ U{0..K}.
    verify_horizon: int = 0
    # Two-stream ShortConv in front of the GDN layer (0 = none): width W over
    # C = 2 Hk dk + Hv dv channels (the q, k and v projections), SiLU.
    conv_width: int = 0

    @property
    def conv_channels(self) -> int:
        return 2 * self.num_qk_heads * self.head_dim_k + self.num_v_heads * self.head_dim_v

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.act_dtype == "bf16" else torch.float32

    @property
    def max_pages(self) -> int:
        return -(-self.prefix_hi // self.page_size)

    def replace(self, **kw) -> "WorkloadSpec":
        d = dict(self.__dict__)
        d.update(kw)
        return WorkloadSpec(**d)


WORKLOADS = {
    "tiny_fp32": WorkloadSpec(
        name="tiny_fp32",
        description="1 request; GDN 2 heads d=64 B=8 fp32; softmax 2q/1kv D=64, prefix 32 "
                    "in 16-token pages; commit at length 5",
        num_requests=1, block_len=8, num_qk_heads=2, num_v_heads=2, head_dim_k=64, head_dim_v=64,
        num_q_heads=2, num_kv_heads=1, head_dim=64, page_size=16, prefix_lo=32, prefix_hi=32,
        act_dtype="f32", denoise_steps=1, accept="fixed", accept_fixed=5, state_prefix_tokens=64,
        seed=0),
    "single_request": WorkloadSpec(
        name="single_request",
        description="1 request; GDN 16 qk / 32 v heads d=128 B=32 bf16; softmax 16q/2kv D=256, "
                    "prefix 4096 in 64-token pages; full-block commit",
        num_requests=1, block_len=32, num_qk_heads=16, num_v_heads=32, head_dim_k=128,
        head_dim_v=128, num_q_heads=16, num_kv_heads=2, head_dim=256, page_size=64,
        prefix_lo=4096, prefix_hi=4096, act_dtype="bf16", denoise_steps=1, accept="full",
        accept_fixed=0, state_prefix_tokens=512, seed=1),
    "serving_batch64": WorkloadSpec(
        name="serving_batch64",
        description="64 requests with single_request shapes, B=32, prefix ~U[512,8192]",
        num_requests=64, block_len=32, num_qk_heads=16, num_v_heads=32, head_dim_k=128,
        head_dim_v=128, num_q_heads=16, num_kv_heads=2, head_dim=256, page_size=64,
        prefix_lo=512, prefix_hi=8192, act_dtype="bf16", denoise_steps=1, accept="full",
        accept_fixed=0, state_prefix_tokens=512, seed=2),
    "small_model_batch256": WorkloadSpec(
        name="small_model_batch256",
        description="256 requests; GDN 16 heads d=128 B=16; softmax 16q/4kv D=128, "
                    "prefix ~U[256,2048]; full-block commit",
        num_requests=256, block_len=16, num_qk_heads=16, num_v_heads=16, head_dim_k=128,
        head_dim_v=128, num_q_heads=16, num_kv_heads=4, head_dim=128, page_size=64,
        prefix_lo=256, prefix_hi=2048, act_dtype="bf16", denoise_steps=1, accept="full",
        accept_fixed=0, state_prefix_tokens=512, seed=3),
    "multistep_batch128": WorkloadSpec(
        name="multistep_batch128",
        description="128 requests with single_request shapes, B=64, 8 denoise steps over a "
                    "prefix ~U[1024,16384], then commit at accept lengths ~U[1,64]",
        num_requests=128, block_len=64, num_qk_heads=16, num_v_heads=32, head_dim_k=128,
        head_dim_v=128, num_q_heads=16, num_kv_heads=2, head_dim=256, page_size=64,
        prefix_lo=1024, prefix_hi=16384, act_dtype="bf16", denoise_steps=8, accept="uniform",
        accept_fixed=0, state_prefix_tokens=512, seed=4),
    "ar_trust_verify_batch64": WorkloadSpec(
        name="ar_trust_verify_batch64",
        description="AR-Trust verify round over serving_batch64's shapes: 64 requests, horizon "
                    "N=16 (block 2N-1 = 31: anchor, K ~ U{0..15} drafts, MASK rows), prefix "
                    "~U[512,8192]; cache-and-scatter commit at accepted offsets ~U{0..K}",
        num_requests=64, block_len=31, num_qk_heads=16, num_v_heads=32, head_dim_k=128,
        head_dim_v=128, num_q_heads=16, num_kv_heads=2, head_dim=256, page_size=64,
        prefix_lo=512, prefix_hi=8192, act_dtype="bf16", denoise_steps=1, accept="full",
        accept_fixed=0, state_prefix_tokens=512, seed=5, verify_horizon=16),
    "shortconv_serving_batch64": WorkloadSpec(
        name="shortconv_serving_batch64",
        description="serving_batch64 with the GDN layer's two-stream ShortConv in front of the "
                    "linear attention: W=4, SiLU, over the 8192 q/k/v channels, conv state "
                    "committed with the recurrent state",
        num_requests=64, block_len=32, num_qk_heads=16, num_v_heads=32, head_dim_k=128,
        head_dim_v=128, num_q_heads=16, num_kv_heads=2, head_dim=256, page_size=64,
        prefix_lo=512, prefix_hi=8192, act_dtype="bf16", denoise_steps=1, accept="full",
        accept_fixed=0, state_prefix_tokens=512, seed=6, conv_width=4),
}


@dataclass
class LinearBlock:
    """Inputs of one gated-delta-rule block: q,k [R,B,Hk,dk], v [R,B,Hv,dv],
    log_decay, beta [R,B,Hv] (fp32)."""
    q: torch.Tensor
    k: torch.Tensor
    v: torch.Tensor
    log_decay: torch.Tensor
    beta: torch.Tensor


@dataclass
class SoftmaxBlock:
    """Block queries q [R,B,Hq,D] and the block's own keys/values [R,B,Hkv,D]."""
    q: torch.Tensor
    k_blk: torch.Tensor
    v_blk: torch.Tensor


@dataclass
class Workload:
    spec: WorkloadSpec
    state_prefix: LinearBlock  # random prefix tokens (q unused) from which S0 is built
    state_pool: torch.Tensor  # [slots, Hv, dk, dv] fp32, NaN everywhere (caller writes S0)
    state_slot: torch.Tensor  # [R] int32, distinct
    denoise: list = field(default_factory=list)  # LinearBlock per denoise step
    commit: LinearBlock = None  # inputs of the token-causal state-update pass
    accept_len: torch.Tensor = None  # [R] int32 in [0, B]
    softmax: list = field(default_factory=list)  # SoftmaxBlock per denoise step
    k_pool: torch.Tensor = None  # [num_pages, Hkv, page_size, D]
    v_pool: torch.Tensor = None
    page_table: torch.Tensor = None  # [R, max_pages] int32, -1 where unused
    prefix_len: torch.Tensor = None  # [R] int32
    verify_len: torch.Tensor = None  # [R] int32, K held drafts (verify workloads)
    verify_accept: torch.Tensor = None  # [R] int32 in [0, K], drafts accepted
    row_type: torch.Tensor = None  # [R, block_len] uint8: 0 for rows 0..K, else 1
    conv_x: list = field(default_factory=list)  # [R,B,C] block inputs of the ShortConv per step
    conv_commit_x: torch.Tensor = None  # [R,B,C] the finalized block (state-update pass)
    conv_state: torch.Tensor = None  # [slots, W-1, C]: last W-1 clean tokens per slot
    conv_weight: torch.Tensor = None  # [C, W] fp32, column i multiplies lag i
    conv_bias: torch.Tensor = None  # [C] fp32


def _l2n(x: torch.Tensor) -> torch.Tensor:
    return x / x.norm(dim=-1, keepdim=True)


def _linear_block(spec, R, B, gen, device, dtype) -> LinearBlock:
    Hk, Hv, dk, dv = spec.num_qk_heads, spec.num_v_heads, spec.head_dim_k, spec.head_dim_v
    f32 = dict(generator=gen, device=device, dtype=torch.float32)
    q = _l2n(torch.randn(R, B, Hk, dk, **f32)).to(dtype)
    k = _l2n(torch.randn(R, B, Hk, dk, **f32)).to(dtype)
    v = torch.randn(R, B, Hv, dv, **f32).to(dtype)
    log_decay = -torch.nn.functional.softplus(torch.randn(R, B, Hv, **f32))
    beta = torch.sigmoid(torch.randn(R, B, Hv, **f32))
    return LinearBlock(q.contiguous(), k.contiguous(), v.contiguous(), log_decay.contiguous(),
                       beta.contiguous())


def generate(spec: WorkloadSpec, device="cpu", *, softmax=True, linear=True) -> Workload:
    """Draw every input of ``spec`` from one generator seeded with ``spec.seed``.

    The draw order is fixed, so the same spec and device give the same tensors."""
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(spec.seed)
    R, B, dtype = spec.num_requests, spec.block_len, spec.torch_dtype
    Hv, dk, dv = spec.num_v_heads, spec.head_dim_k, spec.head_dim_v

    w = Workload(spec=spec, state_prefix=None, state_pool=None, state_slot=None)
    # recurrent-state pool: R used slots at a random permutation of R + spare slots
    nslots = R + spec.spare_slots
    perm = torch.randperm(nslots, generator=gen, device=device)
    w.state_slot = perm[:R].to(torch.int32).contiguous()
    w.state_pool = torch.full((nslots, Hv, dk, dv), float("nan"), device=device,
                              dtype=torch.float32)
    if linear:
        w.state_prefix = _linear_block(spec, R, spec.state_prefix_tokens, gen, device, dtype)
        w.denoise = [_linear_block(spec, R, B, gen, device, dtype)
                     for _ in range(spec.denoise_steps)]
        w.commit = _linear_block(spec, R, B, gen, device, dtype)
    if spec.accept == "full":
        acc = torch.full((R,), B, dtype=torch.int32, device=device)
    elif spec.accept == "fixed":
        acc = torch.full((R,), spec.accept_fixed, dtype=torch.int32, device=device)
    else:
        acc = torch.randint(1, B + 1, (R,), generator=gen, device=device, dtype=torch.int32)
    w.accept_len = acc.contiguous()

    if softmax:
        Hq, Hkv, D, p = spec.num_q_heads, spec.num_kv_heads, spec.head_dim, spec.page_size
        f32 = dict(generator=gen, device=device, dtype=torch.float32)
        lens = torch.randint(spec.prefix_lo, spec.prefix_hi + 1, (R,), generator=gen,
                             device=device, dtype=torch.int32)
        npages = (lens + p - 1) // p
        total = int(npages.sum().item())
        num_pages = total + max(4, math.ceil(0.05 * total))
        page_perm = torch.randperm(num_pages, generator=gen, device=device).to(torch.int32)
        table = torch.full((R, spec.max_pages), -1, dtype=torch.int32, device=device)
        npages_cpu = npages.cpu().tolist()
        off = 0
        for r, n in enumerate(npages_cpu):
            table[r, :n] = page_perm[off:off + n]
            off += n
        k_pool = torch.randn(num_pages, Hkv, p, D, **f32).to(dtype)
        v_pool = torch.randn(num_pages, Hkv, p, D, **f32).to(dtype)
        # poison: spare pages and each request's rows past its prefix end
        valid = torch.zeros(num_pages, p, dtype=torch.bool, device=device)
        lens_cpu = lens.cpu().tolist()
        for r, n in enumerate(npages_cpu):
            if n:
                pages = table[r, :n].long()
                valid[pages] = True
                tail = lens_cpu[r] - (n - 1) * p
                valid[pages[-1], tail:] = False
        bad = ~valid[:, None, :, None].expand(num_pages, Hkv, p, D)
        k_pool.masked_fill_(bad, float("nan"))
        v_pool.masked_fill_(bad, float("nan"))
        w.k_pool, w.v_pool = k_pool.contiguous(), v_pool.contiguous()
        w.page_table, w.prefix_len = table.contiguous(), lens.contiguous()
        for _ in range(spec.denoise_steps):
            qs = torch.randn(R, B, Hq, D, **f32).to(dtype)
            kb = torch.randn(R, B, Hkv, D, **f32).to(dtype)
            vb = torch.randn(R, B, Hkv, D, **f32).to(dtype)
            w.softmax.append(SoftmaxBlock(qs.contiguous(), kb.contiguous(), vb.contiguous()))
    if spec.verify_horizon:
        N = spec.verify_horizon
        if N < 2 or N > B:
            raise ValueError("verify horizon does not fit the block")
        K = torch.randint(0, N, (R,), generator=gen, device=device, dtype=torch.int32)
        u = torch.rand(R, generator=gen, device=device)
        a = torch.minimum((u * (K + 1).float()).floor().to(torch.int32), K)
        w.verify_len, w.verify_accept = K.contiguous(), a.contiguous()
        rows = torch.arange(B, device=device, dtype=torch.int32)
        w.row_type = (rows[None, :] > K[:, None]).to(torch.uint8).contiguous()
    if spec.conv_width:
        W, C = spec.conv_width, spec.conv_channels
        f32 = dict(generator=gen, device=device, dtype=torch.float32)
        w.conv_x = [torch.randn(R, B, C, **f32).to(dtype).contiguous()
                    for _ in range(spec.denoise_steps)]
        w.conv_commit_x = torch.randn(R, B, C, **f32).to(dtype).contiguous()
        nslots = w.state_pool.shape[0]
        cs = torch.randn(nslots, W - 1, C, **f32).to(dtype)
        unused = torch.ones(nslots, dtype=torch.bool, device=device)
        unused[w.state_slot.long()] = False
        cs[unused] = float("nan")
        w.conv_state = cs.contiguous()
        w.conv_weight = (torch.randn(C, W, **f32) / math.sqrt(W)).contiguous()
        w.conv_bias = (0.1 * torch.randn(C, **f32)).contiguous()
    return w


# ---------------------------------------------------------------- training (two-stream)


@dataclass(frozen=True)
class TwoStreamSpec:
    """Two-stream training input of one GDN layer: N sequences of L clean and
    L noisy tokens (the paper's "L = 8192, half clean, half noisy" is
    L = 4096 here), diffusion block B, chunk C of the clean chunkwise pass."""
    name: str
    description: str
    num_seqs: int
    seq_len: int
    block_len: int
    num_qk_heads: int
    num_v_heads: int
    head_dim_k: int
    head_dim_v: int
    act_dtype: str
    seed: int
    chunk_len: int = 64

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.act_dtype == "bf16" else torch.float32

    def replace(self, **kw) -> "TwoStreamSpec":
        d = dict(self.__dict__)
        d.update(kw)
        return TwoStreamSpec(**d)


TWO_STREAM_WORKLOADS = {
    "two_stream_train_b4": TwoStreamSpec(
        name="two_stream_train_b4",
        description="Qwen3.5-2B GDN training shape of the paper's route benchmark: 1 sequence, "
                    "4096 clean + 4096 noisy tokens, 16 heads, d_k = d_v = 128, block B = 4, "
                    "chunk 64",
        num_seqs=1, seq_len=4096, block_len=4, num_qk_heads=16, num_v_heads=16, head_dim_k=128,
        head_dim_v=128, act_dtype="bf16", seed=7),
}


@dataclass
class TwoStreamInput:
    spec: TwoStreamSpec
    clean: LinearBlock  # q unused (the clean outputs are the clean chunkwise pass's)
    noisy: LinearBlock
    S_init: torch.Tensor  # [N, Hv, dk, dv] fp32: the clean state before position 0 (zero)


def generate_two_stream(spec: TwoStreamSpec, device="cpu") -> TwoStreamInput:
    """Clean and noisy token streams with the serving value distributions; the
    clean state before the sequence is zero (a sequence start).  The clean
    chunk states are NOT built here: each caller runs the clean recurrence
    with its own implementation."""
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(spec.seed)
    clean = _linear_block(spec, spec.num_seqs, spec.seq_len, gen, device, spec.torch_dtype)
    noisy = _linear_block(spec, spec.num_seqs, spec.seq_len, gen, device, spec.torch_dtype)
    S0 = torch.zeros(spec.num_seqs, spec.num_v_heads, spec.head_dim_k, spec.head_dim_v,
                     device=device, dtype=torch.float32)
    return TwoStreamInput(spec, clean, noisy, S0)
