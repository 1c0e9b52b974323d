"""flare_block_softmax_attn_noalloc: the softmax call for callers that cannot
allocate device memory (e.g. an engine whose memory manager owns the GPU and
forbids cudaMalloc while serving).  It must give what the workspace-taking
entry point gives, call after call, while drawing its split partials from the
library's own fixed scratch array.  This file is collected last on purpose."""
import numpy as np
import pytest
import torch

from gpu_helpers import OUT_MAX_ABS, OUT_REL_FRO, gen, reduced, rel_fro, softmax_desc
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
def test_noalloc_matches_workspace_entry_point(name):
    spec = W["single_request"] if name == "single_request" else \
        reduced(W["serving_batch64"], 6, 512, 3000)
    w = gen(spec)
    desc = softmax_desc(spec, w)
    ref_out, ref_lse, nb = _with_workspace(w, desc)
    assert 0 < nb <= flare.FLARE_NOALLOC_SCRATCH_BYTES  # the scratch path is exercised
    ref = ref_out.double().cpu().numpy()
    for _ in range(2):  # two calls in a row share the same scratch array
        out, lse = _no_alloc(w, desc)
        got = out.double().cpu().numpy()
        assert np.isfinite(got).all()
        assert np.abs(got - ref).max() <= OUT_MAX_ABS
        assert rel_fro(got, ref) <= OUT_REL_FRO[spec.act_dtype]
        assert (lse - ref_lse).abs().max().item() < LSE_ABS


def test_noalloc_rejects_shapes_beyond_its_scratch():
    spec = W["serving_batch64"]
    w = gen(spec)
    desc = softmax_desc(spec, w)
    nb = flare.flare_softmax_workspace_size(desc)
    if nb <= flare.FLARE_NOALLOC_SCRATCH_BYTES:
        pytest.skip("this shape fits the scratch array on this GPU")
    sb = w.softmax[0]
    out = torch.full_like(sb.q, 3.0)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    rc = flare.flare_block_softmax_attn_noalloc(desc, sb.q, sb.k_blk, sb.v_blk, w.k_pool,
                                                w.v_pool, w.page_table, w.prefix_len, out, None,
                                                st)
    assert rc == flare.FLARE_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert (out == 3.0).all()
