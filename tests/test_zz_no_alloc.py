"""flare_block_softmax_attn_noalloc: the softmax call for callers that cannot
allocate device memory (e.g. an engine whose memory manager owns the GPU and
forbids cudaMalloc while serving).  It must give what the oracle and the
workspace-taking entry point give, call after call, while drawing its split
partials from the library's own fixed scratch array, and it must turn away
shapes whose scratch need exceeds that array.  This file is collected last on
purpose."""
import numpy as np
import pytest
import torch

from gpu_helpers import (OUT_MAX_ABS, OUT_REL_FRO, assert_out_close, gen, oracle_softmax,
                         reduced, rel_fro, softmax_desc)
from paper_2606_01774_gb300 import flare, workloads

pytestmark = pytest.mark.gpu
W = workloads.WORKLOADS
LSE_ABS = 2e-3


def _with_workspace(w, desc):
    sb = w.softmax[0]
    nb = flare.flare_softmax_workspace_size(desc)
    ws = torch.empty(max(nb, 1), dtype=torch.uint8, device="cuda")
    out = torch.empty_like(sb.q)
    lse = torch.empty(sb.q.shape[:3], dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    flare.check(flare.flare_block_softmax_attn(desc, sb.q, sb.k_blk, sb.v_blk, w.k_pool, w.v_pool,
                                               w.page_table, w.prefix_len, out, lse, ws, nb, st))
    assert flare.flare_read_status(st) == (flare.FLARE_OK, 0)
    return out, lse, nb


def _no_alloc(w, desc):
    sb = w.softmax[0]
    out = torch.full_like(sb.q, float("nan"))
    lse = torch.full(sb.q.shape[:3], float("nan"), dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    flare.check(flare.flare_block_softmax_attn_noalloc(desc, sb.q, sb.k_blk, sb.v_blk, w.k_pool,
                                                       w.v_pool, w.page_table, w.prefix_len, out,
                                                       lse, st), "noalloc")
    assert flare.flare_read_status(st) == (flare.FLARE_OK, 0)
    return out, lse


@pytest.mark.parametrize("name", ["single_request", "serving_batch64_r6"])
def test_noalloc_matches_oracle_and_workspace_entry_point(name):
    spec = W["single_request"] if name == "single_request" else \
        reduced(W["serving_batch64"], 6, 512, 3000)
    w = gen(spec)
    desc = softmax_desc(spec, w)
    ref_out, ref_lse, nb = _with_workspace(w, desc)
    assert 0 < nb <= flare.FLARE_NOALLOC_SCRATCH_BYTES  # the scratch path is exercised
    want, want_lse = oracle_softmax(w, 0)
    ref = ref_out.double().cpu().numpy()
    for call in range(2):  # two calls in a row share the same scratch array
        out, lse = _no_alloc(w, desc)
        assert_out_close(out, want, spec.act_dtype, f"{name} call {call} vs oracle")
        assert np.abs(lse.double().cpu().numpy() - want_lse).max() < LSE_ABS
        got = out.double().cpu().numpy()
        assert np.abs(got - ref).max() <= OUT_MAX_ABS
        assert rel_fro(got, ref) <= OUT_REL_FRO[spec.act_dtype]
        assert (lse - ref_lse).abs().max().item() < LSE_ABS


def test_noalloc_rejects_shapes_beyond_its_scratch():
    """A batch of 20 M one-token requests needs ~79 MiB of work-order scratch,
    more than the array holds: the call must return FLARE_ERR_UNSUPPORTED on the
    host, before any launch, so the (small, dummy) tensors it is handed are
    never read or written."""
    R = 20_000_000
    desc = flare.softmax_desc(R, 1, 1, 1, 64, 16, 4, 1, flare.FLARE_DT_BF16, 0.125)
    assert flare.flare_softmax_workspace_size(desc) > flare.FLARE_NOALLOC_SCRATCH_BYTES
    dev = torch.device("cuda")
    q = torch.zeros(64, 64, dtype=torch.bfloat16, device=dev)
    kv = torch.zeros(4, 1, 16, 64, dtype=torch.bfloat16, device=dev)
    table = torch.zeros(64, dtype=torch.int32, device=dev)
    out = torch.full((64, 64), 3.0, dtype=torch.bfloat16, device=dev)
    lse = torch.full((64,), 5.0, dtype=torch.float32, device=dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    rc = flare.flare_block_softmax_attn_noalloc(desc, q, q, q, kv, kv, table, table, out, lse, st)
    assert rc == flare.FLARE_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert (out == 3.0).all() and (lse == 5.0).all()
    assert flare.flare_read_status(st) == (flare.FLARE_OK, 0)
