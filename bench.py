#!/usr/bin/env python3
"""Benchmark of the FLARE block-denoising attention step on GB300.

One step = one pass of the whole hot path over one batch: for each of the
workload's denoise steps, one gated-delta-rule layer call
(flare_block_linear_attn) and one softmax layer call (flare_block_softmax_attn)
over fresh block inputs, then one commit of every request's state at its
accepted length (flare_commit_state).  Metric: block-tokens/s =
requests x block_len x denoise_steps / step time.

Workloads with a ShortConv (--workload shortconv_serving_batch64) add the GDN
layer's two-stream causal ShortConv (flare_short_conv) in front of each linear
call, and its conv-state commit in front of the recurrent-state commit.

The training workload (--workload two_stream_train_b4) times the fused
two-stream forward of one GDN layer (flare_two_stream_fwd) on the paper's
route-benchmark shape; its metric is training tokens/s (clean + noisy).

The AR-Trust verify workload (--workload ar_trust_verify_batch64) times the
verify round instead: flare_verify_linear_attn, flare_block_softmax_attn with
per-request row types, and flare_verify_commit at the accepted offsets; its
block-tokens are requests x block_len per round.

Default workload: multistep_batch128 (128 requests, GDN 16 qk / 32 v heads,
d=128, softmax 16 q / 2 kv heads, D=256, block 64, 8 denoise steps over paged
prefixes ~U[1024,16384], commit at accepted lengths ~U[1,64]).  Each step
streams ~2.7 GB of KV and state (> 129 MB L2), so no L2 flush is needed.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
                  [--impl flare|reference]

Under torchrun (N > 1) every rank runs its own batch (requests are
independent: weak scaling, no collective on the data path); the timed region
is bracketed by barriers and the max over ranks is reported.
``--impl reference`` times the fp64 CPU oracle on a bounded sample of the same
workload on the host cores (rank 0 only).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import shutil
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2606_01774_gb300 import workloads  # noqa: E402

METRIC = "denoise-step attention block-tokens/s"
VERIFY_METRIC = "AR-Trust verify-round attention block-tokens/s"
UNIT = "block-tokens/s"
DEFAULT_WORKLOAD = "multistep_batch128"


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return {"hbm_gbs": pk["hbm_gbs"], "bf16_tflops": pk["bf16_tflops"],
                "bf16_tflops_sustained": pk.get("bf16_tflops_sustained", pk["bf16_tflops"]),
                "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


# ---------------------------------------------------------------- algorithmic counts


def linear_bytes(spec):
    R, B, Hk, Hv, dk, dv = (spec.num_requests, spec.block_len, spec.num_qk_heads,
                            spec.num_v_heads, spec.head_dim_k, spec.head_dim_v)
    e = 2 if spec.act_dtype == "bf16" else 4
    return (R * Hv * dk * dv * 4 + 2 * R * B * Hk * dk * e + R * B * Hv * dv * e
            + 2 * R * B * Hv * 4 + R * B * Hv * dv * e)


def linear_flops(spec):
    B, dk, dv = spec.block_len, spec.head_dim_k, spec.head_dim_v
    per_head = 4 * B * B * dk + 4 * B * dk * dv + 2 * B * B * dv + (2 / 3) * B ** 3
    return spec.num_requests * spec.num_v_heads * per_head


def softmax_bytes(spec, prefix_sum):
    R, B, Hq, Hkv, D = (spec.num_requests, spec.block_len, spec.num_q_heads, spec.num_kv_heads,
                        spec.head_dim)
    e = 2 if spec.act_dtype == "bf16" else 4
    return (2 * prefix_sum * Hkv * D * e + R * B * Hq * D * e + 2 * R * B * Hkv * D * e
            + R * B * Hq * D * e)


def softmax_flops(spec, prefix_sum):
    return 4.0 * spec.block_len * spec.num_q_heads * spec.head_dim * (
        prefix_sum + spec.num_requests * spec.block_len)


def commit_bytes(spec, accept):
    n = int((accept > 0).sum())
    B, Hk, Hv, dk, dv = (spec.block_len, spec.num_qk_heads, spec.num_v_heads, spec.head_dim_k,
                         spec.head_dim_v)
    e = 2 if spec.act_dtype == "bf16" else 4
    R = spec.num_requests
    return (2 * n * Hv * dk * dv * 4 + R * B * Hk * dk * e + R * B * Hv * dv * e
            + 2 * R * B * Hv * 4)


def verify_linear_bytes(spec, verify_len):
    """Verify pass: S0 read, live state written, S^(t) written for t < K, plus
    the block's activations and gates."""
    st = spec.num_v_heads * spec.head_dim_k * spec.head_dim_v * 4
    n_rec = int(np.asarray(verify_len).sum())
    return 2 * spec.num_requests * st + n_rec * st + linear_bytes(spec) - spec.num_requests * st


def verify_linear_flops(spec):
    """fp32 CUDA-core work: per token and head one d_k x d_v product S^T k, one
    rank-one update and one readout, a multiply-add each."""
    return 6.0 * spec.num_requests * spec.num_v_heads * spec.block_len * spec.head_dim_k * \
        spec.head_dim_v


def conv_bytes(spec, commit=False):
    """ShortConv: block in and out, the conv state read (and written on
    commit), filter taps and bias."""
    e = 2 if spec.act_dtype == "bf16" else 4
    R, B, C, W = spec.num_requests, spec.block_len, spec.conv_channels, spec.conv_width
    return 2 * R * B * C * e + R * (W - 1) * C * e * (2 if commit else 1) + C * (W + 1) * 4


def verify_commit_bytes(spec, verify_len, accept):
    st = spec.num_v_heads * spec.head_dim_k * spec.head_dim_v * 4
    n = int((np.asarray(accept) < np.asarray(verify_len)).sum())
    return 2 * n * st


# ---------------------------------------------------------------- ncu traffic


def kernel_of_call(spec):
    """The kernel each layer call of `spec` runs (the library's dispatch: bf16
    128 x 128 states take the persistent denoise kernels -- B <= 32, and 33..64
    as one chunk -- and the tensor-core commit; other shapes the
    one-CTA-per-item kernels)."""
    tc_state = spec.act_dtype == "bf16" and spec.head_dim_k == 128 and spec.head_dim_v == 128
    if tc_state and spec.block_len <= 32:
        linear = "gdr_denoise_persist_kernel"
    elif tc_state and spec.block_len <= 64:
        linear = "gdr_denoise_chunk64_kernel"
    else:
        linear = "gdr_denoise_tc_kernel"
    return {"linear": linear,
            "softmax": "softmax_tc_kernel",
            "commit": "gdr_commit_tc_kernel" if tc_state else "gdr_commit_kernel",
            "shortconv": "short_conv_kernel", "shortconv_commit": "short_conv_kernel"}
VERIFY_KERNEL_OF = {"linear": "gdr_commit_kernel", "softmax": "softmax_tc_kernel",
                    "commit": "verify_commit_kernel"}


def profiled_traffic(kernel, workload):
    """DRAM bytes per launch from the committed ncu summary of `kernel` on
    `workload` (profiles/<kernel>_<workload>_traffic.md), or None when there is
    none or the kernel's source has changed since it was taken."""
    import hashlib

    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload}_traffic.md")
    try:
        fields = {}
        for line in open(path):
            if ":" in line and not line.startswith(" "):
                k, v = line.split(":", 1)
                fields[k.strip()] = v.strip()
        src = os.path.join(ROOT, fields["kernel_source"])
        if hashlib.sha256(open(src, "rb").read()).hexdigest() != fields["kernel_source_sha256"]:
            return None
        return int(fields["traffic_bytes_per_launch"])
    except (OSError, KeyError, ValueError):
        return None


# ---------------------------------------------------------------- clocks


class ClockSampler:
    """nvidia-smi samples every 50 ms while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.proc = None
        self.path = None
        exe = shutil.which("nvidia-smi")
        if exe is None:
            return
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        self.out = open(self.path, "w")
        self.proc = subprocess.Popen(
            [exe, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "50",
             "-i", str(device_index)], stdout=self.out, stderr=subprocess.DEVNULL)

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if "Active" in r[5 + i]
                          and "Not" not in r[5 + i]})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


# ---------------------------------------------------------------- GPU arm


class FlareRunner:
    """Holds one workload on the device and issues the step's C-ABI calls."""

    def __init__(self, spec, device, seed_offset=0):
        from paper_2606_01774_gb300 import flare

        self.flare = flare
        self.spec = spec.replace(seed=spec.seed + seed_offset)
        self.device = device
        self.w = workloads.generate(self.spec, device)
        s = self.spec
        self.act = flare.FLARE_DT_BF16 if s.act_dtype == "bf16" else flare.FLARE_DT_F32
        nslots = self.w.state_pool.shape[0]
        self.ldesc = flare.linear_desc(s.num_requests, s.block_len, s.num_qk_heads,
                                       s.num_v_heads, s.head_dim_k, s.head_dim_v, nslots,
                                       self.act, 1.0 / math.sqrt(s.head_dim_k))
        self.verify = s.verify_horizon > 0
        mode = flare.FLARE_MASK_ROW_TYPE_PER_REQUEST if self.verify else flare.FLARE_MASK_BLOCK_BIDIR
        self.sdesc = flare.softmax_desc(s.num_requests, s.block_len, s.num_q_heads,
                                        s.num_kv_heads, s.head_dim, s.page_size,
                                        self.w.k_pool.shape[0], self.w.page_table.shape[1],
                                        self.act, 1.0 / math.sqrt(s.head_dim), mode,
                                        self.w.row_type if self.verify else None)
        if self.verify:
            self.max_verify = s.verify_horizon - 1
            self.records = torch.empty(s.num_requests, self.max_verify, s.num_v_heads,
                                       s.head_dim_k, s.head_dim_v, device=device)
        self.ws_bytes = flare.flare_softmax_workspace_size(self.sdesc)
        self.ws = torch.empty(max(self.ws_bytes, 256), dtype=torch.uint8, device=device)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)
        self.lin_out = [torch.empty_like(b.v) for b in self.w.denoise]
        self.sm_out = [torch.empty_like(b.q) for b in self.w.softmax]
        self.conv = s.conv_width > 0
        if self.conv:
            self.cdesc = flare.conv_desc(s.num_requests, s.block_len, s.conv_channels,
                                         s.conv_width, self.w.conv_state.shape[0], self.act,
                                         flare.FLARE_ACT_SILU)
            self.conv_out = [torch.empty_like(x) for x in self.w.conv_x]
            self.conv_commit_out = torch.empty_like(self.w.conv_commit_x)
        self.prefill_states()

    def prefill_states(self):
        """Committed state S0 of every request: the gated delta rule over its
        random prefix tokens from the zero state, run through the library's own
        commit in blocks of up to 64 tokens (what a serving prefill does)."""
        fl, s, w = self.flare, self.spec, self.w
        w.state_pool.zero_()
        sp = w.state_prefix
        n = sp.k.shape[1]
        for lo in range(0, n, 64):
            hi = min(lo + 64, n)
            d = fl.linear_desc(s.num_requests, hi - lo, s.num_qk_heads, s.num_v_heads,
                               s.head_dim_k, s.head_dim_v, w.state_pool.shape[0], self.act,
                               1.0 / math.sqrt(s.head_dim_k))
            acc = torch.full((s.num_requests,), hi - lo, dtype=torch.int32, device=self.device)
            fl.check(fl.flare_commit_state(
                d, None, sp.k[:, lo:hi].contiguous(), sp.v[:, lo:hi].contiguous(),
                sp.log_decay[:, lo:hi].contiguous(), sp.beta[:, lo:hi].contiguous(),
                w.state_pool, w.state_slot, acc, None, self.status), "prefill")
        torch.cuda.synchronize()

    def linear(self, i, ev=None):
        fl, w, b = self.flare, self.w, self.w.denoise[i]
        if self.verify:
            rc = fl.flare_verify_linear_attn(self.ldesc, self.max_verify, b.q, b.k, b.v,
                                             b.log_decay, b.beta, w.state_pool, w.state_slot,
                                             w.verify_len, self.lin_out[i], self.records,
                                             self.status)
            if rc:
                fl.check(rc, "flare_verify_linear_attn")
            return
        rc = fl.flare_block_linear_attn(self.ldesc, b.q, b.k, b.v, b.log_decay, b.beta,
                                        w.state_pool, w.state_slot, self.lin_out[i], self.status)
        if rc:
            fl.check(rc, "flare_block_linear_attn")

    def softmax(self, i):
        fl, w, b = self.flare, self.w, self.w.softmax[i]
        rc = fl.flare_block_softmax_attn(self.sdesc, b.q, b.k_blk, b.v_blk, w.k_pool, w.v_pool,
                                         w.page_table, w.prefix_len, self.sm_out[i], None,
                                         self.ws, self.ws_bytes, self.status)
        if rc:
            fl.check(rc, "flare_block_softmax_attn")

    def commit(self):
        fl, w, b = self.flare, self.w, self.w.commit
        if self.verify:
            rc = fl.flare_verify_commit(self.ldesc, self.max_verify, [self.records],
                                        [w.state_pool], w.state_slot, w.verify_accept,
                                        w.verify_len, self.status)
            if rc:
                fl.check(rc, "flare_verify_commit")
            return
        rc = fl.flare_commit_state(self.ldesc, None, b.k, b.v, b.log_decay, b.beta,
                                   w.state_pool, w.state_slot, w.accept_len, None, self.status)
        if rc:
            fl.check(rc, "flare_commit_state")

    def shortconv(self, i):
        """ShortConv of denoise step i's block (i = -1: the state-update pass's
        block, committing the conv state at the accepted lengths)."""
        fl, w = self.flare, self.w
        if i < 0:
            x, out, acc = w.conv_commit_x, self.conv_commit_out, w.accept_len
        else:
            x, out, acc = w.conv_x[i], self.conv_out[i], None
        rc = fl.flare_short_conv(self.cdesc, x, w.conv_state, w.state_slot, w.conv_weight,
                                 w.conv_bias, acc, out, self.status)
        if rc:
            fl.check(rc, "flare_short_conv")

    def _timed(self, events, key, fn, *args):
        if events is None:
            fn(*args)
            return
        events.setdefault(key, []).append(torch.cuda.Event(enable_timing=True))
        events[key][-1].record()
        fn(*args)
        events[key].append(torch.cuda.Event(enable_timing=True))
        events[key][-1].record()

    def step(self, events=None):
        """One pass of the hot path; events (if given) bracket each call."""
        for i in range(self.spec.denoise_steps):
            if self.conv:
                self._timed(events, "shortconv", self.shortconv, i)
            if events is not None:
                events["linear"].append(torch.cuda.Event(enable_timing=True))
                events["linear"][-1].record()
            self.linear(i)
            if events is not None:
                events["linear"].append(torch.cuda.Event(enable_timing=True))
                events["linear"][-1].record()
                events["softmax"].append(torch.cuda.Event(enable_timing=True))
                events["softmax"][-1].record()
            self.softmax(i)
            if events is not None:
                events["softmax"].append(torch.cuda.Event(enable_timing=True))
                events["softmax"][-1].record()
        if self.conv:
            self._timed(events, "shortconv_commit", self.shortconv, -1)
        if events is not None:
            events["commit"].append(torch.cuda.Event(enable_timing=True))
            events["commit"][-1].record()
        self.commit()
        if events is not None:
            events["commit"].append(torch.cuda.Event(enable_timing=True))
            events["commit"][-1].record()


class E2ERunner:
    """The same step through the C ABI with the step's inputs in pinned host
    memory: host->device copies of every per-step input and device->host
    copies of every output happen inside the timed region.  The paged KV pool
    and the recurrent-state pool are the serving caches and stay resident.

    The copies run on their own streams, as a serving loop would issue them:
    every input goes host->device in the order the step consumes it (the
    request metadata, then each denoise step's linear and softmax inputs, then
    the commit's), each layer call waits only for its own inputs, and its
    outputs go device->host as soon as they are written."""

    def __init__(self, fr: FlareRunner):
        self.fr = fr
        w = fr.w
        pin = lambda t: (t.cpu().pin_memory(), t)  # noqa: E731
        meta = (w.page_table, w.prefix_len, w.accept_len, w.state_slot)
        if fr.verify:
            meta = (w.page_table, w.prefix_len, w.state_slot, w.verify_len, w.row_type)
        # groups in consumption order: the metadata, then per denoise step the
        # linear layer's inputs and the softmax layer's, then the commit's
        self.groups = [[pin(t) for t in meta]]
        for i, (b, sb) in enumerate(zip(w.denoise, w.softmax)):
            conv_in = (w.conv_x[i],) if fr.conv else ()
            self.groups.append([pin(t) for t in conv_in + (b.q, b.k, b.v, b.log_decay, b.beta)])
            self.groups.append([pin(t) for t in (sb.q, sb.k_blk, sb.v_blk)])
        if fr.verify:  # the accept decision, known once the round's logits are sampled
            self.groups.append([pin(w.verify_accept)])
        else:
            conv_in = (w.conv_commit_x,) if fr.conv else ()
            self.groups.append([pin(t) for t in conv_in + (w.commit.k, w.commit.v,
                                                           w.commit.log_decay, w.commit.beta)])
        hbuf = lambda d: (d, torch.empty(d.shape, dtype=d.dtype, pin_memory=True))  # noqa: E731
        # per denoise step: the linear layer's outputs (and the ShortConv's),
        # then the softmax layer's
        self.outs = []
        for i, (lo, so) in enumerate(zip(fr.lin_out, fr.sm_out)):
            self.outs.append([hbuf(lo)] + ([hbuf(fr.conv_out[i])] if fr.conv else []))
            self.outs.append([hbuf(so)])
        self.h2d_bytes = sum(h.numel() * h.element_size() for g in self.groups for h, _ in g)
        self.d2h_bytes = sum(h.numel() * h.element_size() for g in self.outs for _, h in g)
        self.s_h2d = torch.cuda.Stream()
        self.s_d2h = torch.cuda.Stream()
        self.ev_in = [torch.cuda.Event() for _ in self.groups]
        self.ev_out = [torch.cuda.Event() for _ in self.outs]

    def step(self):
        fr, cs = self.fr, torch.cuda.current_stream()
        with torch.cuda.stream(self.s_h2d):
            for g, ev in zip(self.groups, self.ev_in):
                for h, d in g:
                    d.copy_(h, non_blocking=True)
                ev.record(self.s_h2d)
        cs.wait_event(self.ev_in[0])

        def send_back(k):  # outputs of group k go to the host as soon as written
            self.ev_out[k].record(cs)
            with torch.cuda.stream(self.s_d2h):
                self.s_d2h.wait_event(self.ev_out[k])
                for d, h in self.outs[k]:
                    h.copy_(d, non_blocking=True)

        for i in range(fr.spec.denoise_steps):
            cs.wait_event(self.ev_in[1 + 2 * i])  # this step's linear inputs
            if fr.conv:
                fr.shortconv(i)
            fr.linear(i)
            send_back(2 * i)
            cs.wait_event(self.ev_in[2 + 2 * i])  # this step's softmax inputs
            fr.softmax(i)
            send_back(2 * i + 1)
        cs.wait_event(self.ev_in[-1])
        if fr.conv:
            fr.shortconv(-1)
        fr.commit()
        self.s_d2h.synchronize()
        cs.synchronize()


TWO_STREAM_METRIC = "two-stream GDR training forward tokens/s"


class TwoStreamRunner:
    """One GDN layer's fused two-stream forward on one training batch.  The
    clean chunk states it consumes (what the clean chunkwise pass hands over)
    are built once by running the library's own exact commit over the clean
    tokens chunk by chunk."""

    def __init__(self, spec, device, seed_offset=0):
        from paper_2606_01774_gb300 import flare

        self.flare = flare
        self.spec = spec.replace(seed=spec.seed + seed_offset)
        self.device = device
        self.x = workloads.generate_two_stream(self.spec, device)
        s, x = self.spec, self.x
        self.act = flare.FLARE_DT_BF16 if s.act_dtype == "bf16" else flare.FLARE_DT_F32
        self.scale = 1.0 / math.sqrt(s.head_dim_k)
        self.desc = flare.two_stream_desc(s.num_seqs, s.seq_len, s.chunk_len, s.block_len,
                                          s.num_qk_heads, s.num_v_heads, s.head_dim_k,
                                          s.head_dim_v, self.act, self.scale)
        n_chunks = s.seq_len // s.chunk_len
        self.chunk_states = torch.empty(s.num_seqs, s.num_v_heads, n_chunks, s.head_dim_k,
                                        s.head_dim_v, device=device)
        self.out = torch.empty_like(x.noisy.v)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)
        self._build_chunk_states()

    def _build_chunk_states(self):
        fl, s, x = self.flare, self.spec, self.x
        pool = x.S_init.clone()
        slot = torch.arange(s.num_seqs, dtype=torch.int32, device=self.device)
        acc = torch.full((s.num_seqs,), s.chunk_len, dtype=torch.int32, device=self.device)
        st = torch.zeros(1, dtype=torch.int32, device=self.device)
        d = fl.linear_desc(s.num_seqs, s.chunk_len, s.num_qk_heads, s.num_v_heads, s.head_dim_k,
                           s.head_dim_v, s.num_seqs, self.act, self.scale)
        c = x.clean
        for ci in range(self.chunk_states.shape[2]):
            self.chunk_states[:, :, ci] = pool
            sl = slice(ci * s.chunk_len, (ci + 1) * s.chunk_len)
            fl.check(fl.flare_commit_state(
                d, None, c.k[:, sl].contiguous(), c.v[:, sl].contiguous(),
                c.log_decay[:, sl].contiguous(), c.beta[:, sl].contiguous(), pool, slot, acc,
                None, st), "chunk states")
        torch.cuda.synchronize()
        assert fl.flare_read_status(st) == (fl.FLARE_OK, 0)

    def step(self, events=None):
        fl, c, n = self.flare, self.x.clean, self.x.noisy
        if events is not None:
            events["two_stream"].append(torch.cuda.Event(enable_timing=True))
            events["two_stream"][-1].record()
        rc = fl.flare_two_stream_fwd(self.desc, self.chunk_states, c.k, c.v, c.log_decay, c.beta,
                                     n.q, n.k, n.v, n.log_decay, n.beta, self.out, self.status)
        if rc:
            fl.check(rc, "flare_two_stream_fwd")
        if events is not None:
            events["two_stream"].append(torch.cuda.Event(enable_timing=True))
            events["two_stream"][-1].record()

    def inputs(self):
        c, n = self.x.clean, self.x.noisy
        return [self.chunk_states, c.k, c.v, c.log_decay, c.beta, n.q, n.k, n.v, n.log_decay,
                n.beta]

    def bytes(self):
        return sum(t.numel() * t.element_size() for t in self.inputs()) + \
            self.out.numel() * self.out.element_size()

    def flops(self):
        """fp32 CUDA-core work per token pair: S^T k (clean), S^T k~, S^T q~ and
        the clean rank-one update, d_k d_v multiply-adds each."""
        s = self.spec
        return 8.0 * s.num_seqs * s.num_v_heads * s.seq_len * s.head_dim_k * s.head_dim_v


def run_two_stream(args, spec, rank, world, local_rank):
    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    from paper_2606_01774_gb300 import flare

    flare.load()
    tr = TwoStreamRunner(spec, device, seed_offset=rank_seed_offset(rank))
    dist = world > 1
    if dist:
        import torch.distributed as tdist
    for _ in range(args.warmup):
        tr.step()
    torch.cuda.synchronize()
    events = {"two_stream": []}
    clocks = ClockSampler(torch.cuda.current_device()) if rank == 0 else None
    if dist:
        tdist.barrier()
    torch.cuda.synchronize()
    launches0 = flare.flare_launch_count()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(args.steps):
        tr.step(events)
    t1.record()
    torch.cuda.synchronize()
    launches = flare.flare_launch_count() - launches0
    if dist:
        tdist.barrier()
    clk = clocks.stop() if clocks else None
    ms_step = max_over_ranks(t0.elapsed_time(t1), dist, device) / args.steps

    e2e_ms, h2d, d2h = None, 0, 0
    if not args.no_e2e:
        pinned = [(t.cpu().pin_memory(), t) for t in tr.inputs()]
        hout = torch.empty(tr.out.shape, dtype=tr.out.dtype, pin_memory=True)
        h2d = sum(h.numel() * h.element_size() for h, _ in pinned)
        d2h = hout.numel() * hout.element_size()

        def e2e_step():
            for h, d in pinned:
                d.copy_(h, non_blocking=True)
            tr.step()
            hout.copy_(tr.out, non_blocking=True)
            torch.cuda.current_stream().synchronize()

        for _ in range(max(1, min(args.warmup, 2))):
            e2e_step()
        if dist:
            tdist.barrier()
        t_e = time.perf_counter()
        for _ in range(args.steps):
            e2e_step()
        e2e_ms = max_over_ranks((time.perf_counter() - t_e) * 1e3 / args.steps, dist, device)
    st, bits = tr.flare.flare_read_status(tr.status)
    if st != tr.flare.FLARE_OK or bits:
        raise RuntimeError(f"two-stream device status {bits:#x}")
    if rank != 0:
        return None
    s = tr.spec
    tokens = 2 * s.num_seqs * s.seq_len
    per = float(np.mean(_elapsed_pairs(events["two_stream"])))
    peaks = load_peaks()
    tc_path = s.act_dtype == "bf16" and s.head_dim_k == 128 and s.head_dim_v == 128
    if tc_path:
        # bf16 activations: the chunk's products run as bf16 tensor-core MMAs
        # (kind::f16); peak = the measured bf16 burst rate
        peak = peaks["bf16_tflops"]
        peak_source = f"{peaks['source']} (bf16_tflops)"
        bound = "tensor"
    else:
        mhz = (clk or {}).get("sm_mhz") or 1920.0
        peak = 152 * 128 * 2 * mhz * 1e6 / 1e12
        peak_source = "fp32 CUDA-core count x median SM clock"
        bound = "alu"
    t_cmp = tr.flops() / (peak * 1e12)
    t_hbm = tr.bytes() / (peaks["hbm_gbs"] * 1e9)
    if t_cmp > t_hbm:
        roof = {"bound": bound, "achieved": tr.flops() / (per / 1e3) / 1e12, "peak": peak,
                "unit": "TFLOP/s", "peak_source": peak_source,
                "algorithmic_per_launch": tr.flops()}
    else:
        roof = {"bound": "hbm", "achieved": tr.bytes() / (per / 1e3) / 1e9,
                "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "peak_source": f"{peaks['source']} (hbm_gbs)",
                "algorithmic_per_launch": tr.bytes()}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["traffic"] = profiled_traffic("two_stream_chunk_kernel" if tc_path else "two_stream_fwd_kernel",
                                       s.name)
    roof["kernel"] = "flare_two_stream_fwd"
    return {
        "metric": TWO_STREAM_METRIC, "value": world * tokens / (ms_step / 1e3),
        "unit": "tokens/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": s.act_dtype, "data": "synthetic",
        "config": {"workload": s.name, "sequences": s.num_seqs, "clean_tokens": s.seq_len,
                   "noisy_tokens": s.seq_len, "block_len": s.block_len,
                   "chunk_len": s.chunk_len, "heads": [s.num_qk_heads, s.num_v_heads],
                   "head_dim": [s.head_dim_k, s.head_dim_v], "parallelism": f"replicas{world}",
                   "l2": f"no flush: each step reads {tr.bytes() / 1e6:.0f} MB > 129 MB L2",
                   "context": "paper, one A100-80GB: Route II forward 17.64 ms at B = 4 "
                              "(clean chunkwise pass included)"},
        "per_call_ms": {"two_stream": per},
        "roofline": roof,
        "e2e": None if e2e_ms is None else {
            "value": world * tokens / (e2e_ms / 1e3), "unit": "tokens/s", "ms_per_step": e2e_ms,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": int(launches),
        "clocks": clk,
    }


def two_stream_oracle_rate(spec, seed_offset=0):
    """The fp64 oracle on the whole training sequence (every head), drawn on
    the host with the same recipe, wall-timed."""
    import oracle

    oracle.build()
    sub = spec.replace(seed=spec.seed + seed_offset)
    x = workloads.generate_two_stream(sub, "cpu")
    c, n = x.clean, x.noisy
    t0 = time.perf_counter()
    res = oracle.two_stream_fwd((c.k, c.v, c.log_decay, c.beta),
                                (n.q, n.k, n.v, n.log_decay, n.beta), x.S_init, sub.block_len,
                                sub.chunk_len)
    secs = time.perf_counter() - t0
    assert np.isfinite(res["out"]).all()
    tokens = 2 * spec.num_seqs * spec.seq_len
    desc = (f"{spec.name} ({spec.seq_len} clean + {spec.seq_len} noisy tokens, "
            f"{spec.num_v_heads} heads, drawn on the host with the same recipe), wall time "
            f"measured; the oracle's loop runs over (sequence, head) items")
    return tokens / secs, secs, oracle.max_threads(), desc


def max_over_ranks(x, distributed, device):
    """Max of a per-rank scalar over all ranks (timing only: no data-path collective)."""
    if not distributed:
        return x
    import torch.distributed as tdist

    t = torch.tensor([x], dtype=torch.float64, device=device)
    tdist.all_reduce(t, op=tdist.ReduceOp.MAX)
    return float(t.item())


def rank_seed_offset(rank):
    """Each rank draws its own batch (independent requests: weak scaling)."""
    return 1000 * rank


def _elapsed_pairs(evs):
    return [evs[i].elapsed_time(evs[i + 1]) for i in range(0, len(evs), 2)]


SUSTAINED_AFTER_S = 2.0  # timed regions at least this long use the sustained tensor peak


def tensor_peak(peaks, timed_s):
    """The measured bf16 peak that applies to a kernel timed inside a region of
    timed_s seconds: the burst figure for short regions, the sustained
    (power-capped) one for regions of seconds."""
    key = "bf16_tflops_sustained" if timed_s >= SUSTAINED_AFTER_S else "bf16_tflops"
    return peaks[key], key


def _warm_up(fr, warmup, clocks_rank0=False):
    """Untimed warm-up steps; returns the per-call event lists to fill and the
    clock sampler (rank 0) started just before the timed region."""
    flare = fr.flare
    for _ in range(warmup):
        fr.step()
    torch.cuda.synchronize()
    st, bits = flare.flare_read_status(fr.status)
    if st != flare.FLARE_OK:
        raise RuntimeError(f"device status {bits:#x} after warm-up")
    events = {"linear": [], "softmax": [], "commit": []}
    if fr.conv:
        events.update(shortconv=[], shortconv_commit=[])
    clocks = ClockSampler(torch.cuda.current_device()) if clocks_rank0 else None
    return events, clocks


def summarise(fr, per, timed_s, clk):
    """Algorithmic bytes and flops of each call, the step's achieved HBM
    bandwidth and the roofline of the dominant kernel."""
    s = fr.spec
    prefix_sum = int(fr.w.prefix_len.sum().item())
    acc = fr.w.accept_len.cpu().numpy()
    peaks = load_peaks()
    kern = {
        "linear": dict(bytes=linear_bytes(s), flops=linear_flops(s), kernel="flare_block_linear_attn"),
        "softmax": dict(bytes=softmax_bytes(s, prefix_sum), flops=softmax_flops(s, prefix_sum),
                        kernel="flare_block_softmax_attn"),
        "commit": dict(bytes=commit_bytes(s, acc), flops=0.0, kernel="flare_commit_state"),
    }
    if fr.verify:
        vl, va = fr.w.verify_len.cpu().numpy(), fr.w.verify_accept.cpu().numpy()
        kern["linear"] = dict(bytes=verify_linear_bytes(s, vl), flops=verify_linear_flops(s),
                              kernel="flare_verify_linear_attn", fp32_alu=True)
        kern["commit"] = dict(bytes=verify_commit_bytes(s, vl, va), flops=0.0,
                              kernel="flare_verify_commit")
    if fr.conv:
        kern["shortconv"] = dict(bytes=conv_bytes(s), flops=0.0, kernel="flare_short_conv")
        kern["shortconv_commit"] = dict(bytes=conv_bytes(s, commit=True), flops=0.0,
                                        kernel="flare_short_conv")
    once = ("commit", "shortconv_commit")
    share = {k: per[k] * (s.denoise_steps if k not in once else 1) for k in per}
    dom = max(share, key=share.get)
    kd = kern[dom]
    dur_s = per[dom] / 1e3
    tc_peak, tc_key = tensor_peak(peaks, timed_s)
    t_hbm = kd["bytes"] / (peaks["hbm_gbs"] * 1e9)
    t_tc = kd["flops"] / (tc_peak * 1e12)
    if kd.get("fp32_alu"):
        # CUDA-core fp32: 152 SMs x 128 lanes x 2 flops x the median SM clock
        mhz = (clk or {}).get("sm_mhz") or 1920.0
        alu_peak = 152 * 128 * 2 * mhz * 1e6 / 1e12
        t_tc = kd["flops"] / (alu_peak * 1e12)
    if kd.get("fp32_alu") and t_tc > t_hbm:
        roof = {"bound": "alu", "achieved": kd["flops"] / dur_s / 1e12, "peak": alu_peak,
                "unit": "TFLOP/s"}
        peak_source = "fp32 CUDA-core count x median SM clock"
    elif t_tc > t_hbm:
        roof = {"bound": "tensor", "achieved": kd["flops"] / dur_s / 1e12, "peak": tc_peak,
                "unit": "TFLOP/s"}
        peak_source = f"{peaks['source']} ({tc_key}; timed region {timed_s:.2f} s)"
    else:
        roof = {"bound": "hbm", "achieved": kd["bytes"] / dur_s / 1e9,
                "peak": peaks["hbm_gbs"], "unit": "GB/s"}
        peak_source = f"{peaks['source']} (hbm_gbs)"
    roof["frac"] = roof["achieved"] / roof["peak"]
    kernel_of = VERIFY_KERNEL_OF if fr.verify else kernel_of_call(s)
    roof["traffic"] = profiled_traffic(kernel_of[dom], s.name) if dom in kernel_of else None
    roof["kernel"] = kd["kernel"]
    roof["peak_source"] = peak_source
    roof["algorithmic_per_launch"] = kd["flops"] if roof["bound"] == "tensor" else kd["bytes"]
    step_bytes = sum(kd_["bytes"] * (1 if k in once else s.denoise_steps)
                     for k, kd_ in kern.items())
    per_call_gbs = {k: kern[k]["bytes"] / (per[k] / 1e3) / 1e9 for k in per}
    return kern, roof, step_bytes, per_call_gbs


def run_steps(fr, steps, warmup, dist=False, device=None, clocks_rank0=False):
    """Times `steps` steps of a FlareRunner; returns (per-call mean ms, total
    ms, launches, clock record)."""
    flare = fr.flare
    events, clocks = _warm_up(fr, warmup, clocks_rank0)
    if dist:
        import torch.distributed as tdist

        tdist.barrier()
    torch.cuda.synchronize()
    launches0 = flare.flare_launch_count()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(steps):
        fr.step(events)
    t1.record()
    torch.cuda.synchronize()
    launches = flare.flare_launch_count() - launches0
    if dist:
        tdist.barrier()
    clk = clocks.stop() if clocks else None
    ms = max_over_ranks(t0.elapsed_time(t1), dist, device)
    per = {k: float(np.mean(_elapsed_pairs(v))) for k, v in events.items()}
    return per, ms, launches, clk


PER_CONFIG_WORKLOADS = ("serving_batch64", "small_model_batch256")


def run_per_config(steps, warmup, device, names=PER_CONFIG_WORKLOADS):
    """The other batched workloads, timed in the same process after the
    headline one: ms per step, per-call ms and GB/s, the step's achieved HBM
    bandwidth and the dominant kernel's roofline."""
    out = {}
    for name in names:
        fr = FlareRunner(workloads.WORKLOADS[name], device)
        per, ms, launches, _ = run_steps(fr, steps, warmup)
        ms_step = ms / steps
        kern, roof, step_bytes, gbs = summarise(fr, per, ms / 1e3, None)
        s = fr.spec
        peaks = load_peaks()
        st, bits = fr.flare.flare_read_status(fr.status)
        if st != fr.flare.FLARE_OK:
            raise RuntimeError(f"{name}: device status {bits:#x}")
        out[name] = {
            "value": s.num_requests * s.block_len * s.denoise_steps / (ms_step / 1e3),
            "unit": UNIT, "ms_per_step": ms_step, "steps": steps,
            "achieved_hbm_gbs": step_bytes / (ms_step / 1e3) / 1e9,
            "step_hbm_frac": step_bytes / (ms_step / 1e3) / 1e9 / peaks["hbm_gbs"],
            "step_bytes": step_bytes, "per_call_ms": per, "per_call_gbs": gbs,
            "per_call_hbm_frac": {k: v / peaks["hbm_gbs"] for k, v in gbs.items()},
            "roofline": roof, "gpu_launches": int(launches),
        }
        del fr
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
    return out


def run_flare(args, spec, rank, world, local_rank):
    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    from paper_2606_01774_gb300 import flare

    flare.load()
    fr = FlareRunner(spec, device, seed_offset=rank_seed_offset(rank))
    dist = world > 1
    if dist:
        import torch.distributed as tdist

    per, ms, launches, clk = run_steps(fr, args.steps, args.warmup, dist, device,
                                       clocks_rank0=rank == 0)
    ms_step = ms / args.steps

    # end-to-end through host buffers
    e2e, e2e_ms = None, None
    if not args.no_e2e:
        e2e = E2ERunner(fr)
        for _ in range(max(1, min(args.warmup, 2))):
            e2e.step()
        if dist:
            tdist.barrier()
        t_e = time.perf_counter()
        for _ in range(args.steps):
            e2e.step()
        e2e_ms = max_over_ranks((time.perf_counter() - t_e) * 1e3 / args.steps, dist, device)
    st, bits = flare.flare_read_status(fr.status)
    if st != flare.FLARE_OK:
        raise RuntimeError(f"device status {bits:#x} after timing")

    if rank != 0:
        return None
    s = fr.spec
    tokens = s.num_requests * s.block_len * s.denoise_steps
    value = world * tokens / (ms_step / 1e3)
    kern, roof, step_bytes, per_call_gbs = summarise(fr, per, ms / 1e3, clk)
    s_extra = {}
    if fr.verify:
        s_extra = {"verify_horizon": s.verify_horizon,
                   "verify_len_mean": float(fr.w.verify_len.float().mean())}
    if fr.conv:
        s_extra = {"shortconv": {"width": s.conv_width, "channels": s.conv_channels,
                                 "activation": "silu"}}
    line = {
        "metric": METRIC if not fr.verify else VERIFY_METRIC, "value": value, "unit": UNIT,
        "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": s.act_dtype, "data": "synthetic",
        "config": {"workload": s.name, "requests": s.num_requests, "block_len": s.block_len,
                   "denoise_steps": s.denoise_steps, "gdn_heads": [s.num_qk_heads, s.num_v_heads],
                   "head_dim_k": s.head_dim_k, "softmax_heads": [s.num_q_heads, s.num_kv_heads],
                   "head_dim": s.head_dim, "page_size": s.page_size,
                   "prefix": [s.prefix_lo, s.prefix_hi], "parallelism": f"replicas{world}",
                   "l2": f"no flush: each step streams {step_bytes / 1e9:.2f} GB > 129 MB L2",
                   **s_extra},
        "achieved_hbm_gbs": step_bytes / (ms_step / 1e3) / 1e9,
        "per_call_ms": per,
        "per_call_gbs": per_call_gbs,
        "roofline": roof,
        "e2e": None if e2e is None else {
            "value": world * tokens / (e2e_ms / 1e3), "unit": UNIT, "ms_per_step": e2e_ms,
            "h2d_bytes_per_step": e2e.h2d_bytes, "d2h_bytes_per_step": e2e.d2h_bytes},
        "gpu_launches": int(launches),
        "clocks": clk,
    }
    if world == 1 and not args.no_per_config and s.name == DEFAULT_WORKLOAD:
        del e2e
        del fr
        torch.cuda.empty_cache()
        line["per_config"] = run_per_config(args.steps, args.warmup, device)
    return line


# ---------------------------------------------------------------- oracle (CPU) arm


def oracle_sample_rate(spec, n_requests, seed_offset=0):
    """Times the fp64 oracle on a bounded sample of the workload (drawn on the
    host with the same recipe): the first n_requests with every head, the
    workload's whole step for them (each denoise step's linear and softmax
    layer calls, with the ShortConv where the workload has one, then the
    commit), timed end to end with the wall clock.  Returns (block-tokens/s,
    measured seconds, threads, sample description)."""
    import oracle

    oracle.build()
    sub = spec.replace(num_requests=n_requests, seed=spec.seed + seed_offset)
    w = workloads.generate(sub, "cpu")
    R, Hv, dk, dv = sub.num_requests, sub.num_v_heads, sub.head_dim_k, sub.head_dim_v
    c, sp = w.commit, w.state_prefix
    S0 = oracle.gdr_per_token(None, sp.k, sp.v, sp.log_decay, sp.beta,
                              np.zeros((1, Hv, dk, dv), np.float32),
                              np.zeros(R, np.int32), None, blockend=False)["state"]
    pool = S0.astype(np.float32)
    slots = np.arange(R, dtype=np.int32)
    scale = 1.0 / math.sqrt(sub.head_dim)
    t0 = time.perf_counter()
    if spec.verify_horizon:
        # AR-Trust verify round: verify pass, per-row-type softmax, commit
        mv = spec.verify_horizon - 1
        b, sb = w.denoise[0], w.softmax[0]
        o = oracle.gdr_verify(b.q, b.k, b.v, b.log_decay, b.beta, pool, slots, w.verify_len, mv)
        oracle.block_softmax(sb.q, sb.k_blk, sb.v_blk, w.k_pool, w.v_pool, w.page_table,
                             w.prefix_len, scale=scale, mask_mode=3, row_type=w.row_type)
        live = pool.astype(np.float64)
        live[slots] = o["state"]
        oracle.verify_commit([o["records"]], [live], slots, w.verify_accept, w.verify_len)
    else:
        for i in range(sub.denoise_steps):
            b, sb = w.denoise[i], w.softmax[i]
            if spec.conv_width:
                oracle.short_conv(w.conv_x[i], w.conv_state, slots_conv(w), w.conv_weight,
                                  w.conv_bias)
            oracle.gdr_per_token(b.q, b.k, b.v, b.log_decay, b.beta, pool, slots, None,
                                 state=False)
            oracle.block_softmax(sb.q, sb.k_blk, sb.v_blk, w.k_pool, w.v_pool, w.page_table,
                                 w.prefix_len, scale=scale)
        if spec.conv_width:
            oracle.short_conv(w.conv_commit_x, w.conv_state, slots_conv(w), w.conv_weight,
                              w.conv_bias, accept_len=w.accept_len)
        oracle.gdr_per_token(None, c.k, c.v, c.log_decay, c.beta, pool, slots, w.accept_len,
                             blockend=False)
    secs = time.perf_counter() - t0
    tokens = R * spec.block_len * spec.denoise_steps
    what = ("the verify pass, the softmax with per-row types and the commit"
            if spec.verify_horizon else
            f"{spec.denoise_steps} denoise step(s) (linear + softmax"
            + (" + ShortConv" if spec.conv_width else "") + ") and the commit")
    desc = (f"{R} request(s) of {spec.name} drawn on the host with the same recipe "
            f"(prefix {int(w.prefix_len.sum())} tokens), all heads: {what}, wall time "
            f"measured; the oracle's loops run over (request, head) and (request, head, row) "
            f"items, at least {R * min(Hv, sub.num_q_heads * sub.block_len)} per call")
    return tokens / secs, secs, oracle.max_threads(), desc


def slots_conv(w):
    return w.state_slot.cpu().numpy().astype(np.int32)


def run_reference(args, spec):
    """The oracle arm: every step is one request of the workload (a fresh
    seeded draw per step), its whole step on the host cores, wall-timed."""
    secs = []
    threads, desc, prefix = None, None, []
    for i in range(args.warmup + args.steps):
        _, sec, threads, desc = oracle_sample_rate(spec, 1, seed_offset=i)
        if i >= args.warmup:
            secs.append(sec)
    tokens = spec.block_len * spec.denoise_steps
    value = len(secs) * tokens / sum(secs)
    return {
        "impl": "reference", "metric": METRIC if not spec.verify_horizon else VERIFY_METRIC,
        "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * float(np.mean(secs)),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": spec.name, "requests_per_step": 1,
                   "block_tokens_per_step": tokens, "parallelism": "host cores"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": "each step: " + desc,
                         "seconds_timed": float(sum(secs))},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=40)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD,
                    choices=sorted(workloads.WORKLOADS) + sorted(workloads.TWO_STREAM_WORKLOADS))
    ap.add_argument("--impl", default="flare", choices=["flare", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true",
                    help="skip the host-buffer end-to-end measurement (profiling runs)")
    ap.add_argument("--cpu-sample-requests", type=int, default=2)
    ap.add_argument("--no-per-config", action="store_true",
                    help="skip timing the other batched workloads after the headline one")
    ap.add_argument("--requests", type=int, default=0,
                    help="profiling cut: the workload's shapes with this many requests "
                         "(its line is no bench value)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "flare":
        ap.error("--warmup must be >= 3")
    training = args.workload in workloads.TWO_STREAM_WORKLOADS
    spec = (workloads.TWO_STREAM_WORKLOADS if training else workloads.WORKLOADS)[args.workload]
    if args.requests > 0 and not training:
        spec = spec.replace(num_requests=args.requests)
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return 0
        if training:
            secs = [two_stream_oracle_rate(spec, i)[1] for i in range(args.warmup + args.steps)]
            rate, _, threads, desc = two_stream_oracle_rate(spec, 0)
            secs = secs[args.warmup:]
            value = len(secs) * 2 * spec.num_seqs * spec.seq_len / sum(secs)
            print(json.dumps({
                "impl": "reference", "metric": TWO_STREAM_METRIC, "value": value,
                "unit": "tokens/s", "n_gpus": args.gpus, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": 1e3 * float(np.mean(secs)),
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                "data": "synthetic",
                "config": {"workload": spec.name, "parallelism": "host cores"},
                "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": threads,
                                 "kind": "oracle", "sample": "each step: " + desc},
                "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}), flush=True)
            return 0
        print(json.dumps(run_reference(args, spec)), flush=True)
        return 0

    if world > 1:
        import torch.distributed as tdist

        torch.cuda.set_device(local_rank)
        tdist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    if training:
        line = run_two_stream(args, spec, rank, world, local_rank)
        if rank == 0:
            if world == 1 and not args.no_cpu_baseline:
                rate, secs, threads, desc = two_stream_oracle_rate(spec)
                line["cpu_baseline"] = {"value": rate, "unit": "tokens/s", "cores": threads,
                                        "kind": "oracle", "sample": desc,
                                        "seconds_measured": secs}
            print(json.dumps(line), flush=True)
        if world > 1:
            tdist.destroy_process_group()
        return 0
    line = run_flare(args, spec, rank, world, local_rank)
    if rank == 0:
        if world == 1 and not args.no_cpu_baseline:
            rate, secs, threads, desc = oracle_sample_rate(spec, args.cpu_sample_requests)
            line["cpu_baseline"] = {"value": rate, "unit": UNIT, "cores": threads,
                                    "kind": "oracle", "sample": desc, "seconds_measured": secs}
        print(json.dumps(line), flush=True)
    if world > 1:
        tdist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
