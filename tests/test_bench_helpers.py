"""Host-side checks of the benchmark's roofline plumbing (no GPU): the peak a
tensor-bound kernel is measured against, the kernel each layer call runs, the
DRAM traffic read from the committed ncu summaries, and the algorithmic byte
counts against the sizes of the tensors the workload generator draws."""
import glob
import os
import shutil

import pytest
import torch

import bench
from paper_2606_01774_gb300 import workloads

W = workloads.WORKLOADS


def test_tensor_peak_is_burst_for_short_regions_and_sustained_for_long_ones():
    peaks = {"bf16_tflops": 1885.3, "bf16_tflops_sustained": 1689.0}
    assert bench.tensor_peak(peaks, 0.37) == (1885.3, "bf16_tflops")
    assert bench.tensor_peak(peaks, bench.SUSTAINED_AFTER_S - 1e-3) == (1885.3, "bf16_tflops")
    assert bench.tensor_peak(peaks, bench.SUSTAINED_AFTER_S) == (1689.0, "bf16_tflops_sustained")


@pytest.mark.parametrize("name,linear,commit", [
    ("serving_batch64", "gdr_denoise_persist_kernel", "gdr_commit_tc_kernel"),      # B = 32
    ("small_model_batch256", "gdr_denoise_persist_kernel", "gdr_commit_tc_kernel"),  # B = 16
    ("multistep_batch128", "gdr_denoise_chunk64_kernel", "gdr_commit_tc_kernel"),   # B = 64
    ("tiny_fp32", "gdr_denoise_tc_kernel", "gdr_commit_kernel"),                     # fp32, d = 64
])
def test_kernel_of_call_follows_the_dispatch(name, linear, commit):
    k = bench.kernel_of_call(W[name])
    assert k["linear"] == linear and k["commit"] == commit
    assert k["softmax"] == "softmax_tc_kernel"


def _traffic_summaries():
    names = sorted(set(W) | set(workloads.TWO_STREAM_WORKLOADS), key=len, reverse=True)
    out = []
    for path in sorted(glob.glob(os.path.join(bench.ROOT, "profiles", "*_traffic.md"))):
        base = os.path.basename(path)[: -len("_traffic.md")]
        wl = next((n for n in names if base.endswith("_" + n)), None)
        if wl is not None:
            out.append((base[: -len(wl) - 1], wl, path))
    return out


def _field(path, key):
    for line in open(path):
        if line.startswith(key + ":"):
            return line.split(":", 1)[1].strip()
    return None


def test_every_committed_traffic_summary_is_read_back():
    found = _traffic_summaries()
    assert found, "no traffic summaries under profiles/"
    for kernel, wl, path in found:
        got = bench.profiled_traffic(kernel, wl)
        assert got == int(_field(path, "traffic_bytes_per_launch")), (kernel, wl)


def test_profiled_traffic_is_none_for_a_changed_source_or_a_missing_summary(tmp_path, monkeypatch):
    kernel, wl, path = _traffic_summaries()[0]
    src = _field(path, "kernel_source")
    (tmp_path / "profiles").mkdir()
    shutil.copy(path, tmp_path / "profiles" / os.path.basename(path))
    os.makedirs(tmp_path / os.path.dirname(src))
    shutil.copy(os.path.join(bench.ROOT, src), tmp_path / src)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.profiled_traffic(kernel, wl) is not None  # an unchanged copy still matches
    with open(tmp_path / src, "a") as f:
        f.write("\n// changed\n")
    assert bench.profiled_traffic(kernel, wl) is None
    assert bench.profiled_traffic(kernel, "no_such_workload") is None


def _nbytes(*ts):
    return sum(t.numel() * t.element_size() for t in ts)


@pytest.mark.parametrize("name", ["serving_batch64", "multistep_batch128", "tiny_fp32"])
def test_linear_bytes_are_the_call_tensors(name):
    # one request's worth of the workload: state read once, block activations
    # and gates read, the block-end output written (same shape as v)
    spec = W[name].replace(num_requests=2)
    w = workloads.generate(spec, softmax=False)
    blk = w.denoise[0]
    states = spec.num_requests * spec.num_v_heads * spec.head_dim_k * spec.head_dim_v * 4
    want = states + _nbytes(blk.q, blk.k, blk.v, blk.log_decay, blk.beta) + _nbytes(blk.v)
    assert bench.linear_bytes(spec) == want


@pytest.mark.parametrize("name", ["serving_batch64", "small_model_batch256"])
def test_softmax_bytes_are_the_call_tensors(name):
    # the prefix keys and values read once, block queries, keys and values read,
    # the output written (same shape as q)
    spec = W[name].replace(num_requests=3)
    w = workloads.generate(spec, linear=False)
    sb = w.softmax[0]
    P = int(w.prefix_len.sum())
    e = w.k_pool.element_size()
    kv = 2 * P * spec.num_kv_heads * spec.head_dim * e
    want = kv + _nbytes(sb.q, sb.k_blk, sb.v_blk) + _nbytes(sb.q)
    assert bench.softmax_bytes(spec, P) == want


def test_softmax_flops_count_both_products():
    # S = Q K^T and O = P V over the prefix and the block's own keys: 2 flops per
    # multiply-add, two products
    spec = W["serving_batch64"].replace(num_requests=2)
    P = 1000
    keys = P + spec.num_requests * spec.block_len
    rows_per_key = spec.block_len * spec.num_q_heads
    assert bench.softmax_flops(spec, P) == 2 * 2 * rows_per_key * spec.head_dim * keys


def test_commit_bytes_skip_requests_that_commit_nothing():
    spec = W["serving_batch64"].replace(num_requests=4)
    st = spec.num_v_heads * spec.head_dim_k * spec.head_dim_v * 4
    acc = torch.tensor([0, 3, 32, 0]).numpy()
    none = bench.commit_bytes(spec, torch.zeros(4, dtype=torch.int64).numpy())
    assert bench.commit_bytes(spec, acc) - none == 2 * 2 * st
