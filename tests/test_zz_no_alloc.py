"""The decode entry point that allocates nothing (padoc_branch_decode_attn_noalloc).

It serves callers that cannot allocate device memory themselves: a plugin inside a framework that
owns all device memory, or a latency-critical decode loop that must not call cudaMalloc. Its
split-K partials live in the library's fixed device array. This file is collected last so that a
run stopping at the first failure has run every other test first; it passes alone in a fresh
process and after the other tests.
"""
import math

import numpy as np
import pytest
import torch

from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import inputs
from paper_2608_06146_gb300 import padoc_attn as pa
from paper_2608_06146_gb300.engine import DecodePlan

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
O_TOL, LSE_TOL = 1.5e-2, 1e-3   # the bf16 decode tolerances of the parity tests


def test_noalloc_decode_matches_workspace_decode_on_two_calls():
    pbuild.build()
    pa.load_library()
    wl = inputs.dense_page()                      # 64 branches on one page
    di = inputs.decode_inputs(wl, 21)
    plan = DecodePlan(wl.pages, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, DEV)
    assert pa.padoc_decode_workspace_size(plan.info) <= pa.PADOC_STATIC_WORKSPACE_BYTES
    S = plan.num_streams
    k_pool, v_pool = di.k_pool.to(DEV), di.v_pool.to(DEV)
    pt, st = torch.from_numpy(di.page_table).to(DEV), torch.from_numpy(di.stream_table).to(DEV)
    scale = 1.0 / math.sqrt(wl.head_dim)
    g = torch.Generator().manual_seed(77)
    queries = [di.q.to(DEV), torch.randn(di.q.shape, generator=g).to(torch.bfloat16).to(DEV)]
    for call, q in enumerate(queries):            # two calls in a row, different queries
        ref_o = torch.empty((S, 16, 128), dtype=torch.bfloat16, device=DEV)
        ref_l = torch.empty((S, 16), dtype=torch.float32, device=DEV)
        plan.run(k_pool, v_pool, pt, st, q, scale, ref_o, ref_l)
        out = torch.full((S, 16, 128), float("nan"), dtype=torch.bfloat16, device=DEV)
        lse = torch.full((S, 16), float("nan"), dtype=torch.float32, device=DEV)
        pa.padoc_branch_decode_attn_noalloc(k_pool, v_pool, plan.info, plan.plan_dev, pt, st, q, scale, out, lse)
        pa.padoc_check_device_errors()
        do = (out.float() - ref_o.float()).abs().max().item()
        dl = (lse - ref_l).abs().max().item()
        assert math.isfinite(do) and do <= O_TOL, f"call {call}: max |dO| = {do}"
        assert math.isfinite(dl) and dl <= LSE_TOL, f"call {call}: max |dLSE| = {dl}"


def test_noalloc_rejects_a_plan_beyond_the_array():
    pa.load_library()
    wl = inputs.serving_batch(num_pages=128)      # its split-K partials need more than 32 MiB
    plan = DecodePlan(wl.pages, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, DEV)
    assert pa.padoc_decode_workspace_size(plan.info) > pa.PADOC_STATIC_WORKSPACE_BYTES
    S = plan.num_streams
    dummy_pool = torch.zeros((1, 2, 16, 128), dtype=torch.bfloat16, device=DEV)
    table = torch.zeros((max(len(wl.pages), 1), plan.info.max_page_blocks), dtype=torch.int32, device=DEV)
    stable = torch.zeros((S, max(plan.info.max_stream_blocks, 1)), dtype=torch.int32, device=DEV)
    q = torch.zeros((S, 16, 128), dtype=torch.bfloat16, device=DEV)
    out, lse = torch.empty_like(q), torch.empty((S, 16), dtype=torch.float32, device=DEV)
    with pytest.raises(pa.PadocError) as e:
        pa.padoc_branch_decode_attn_noalloc(dummy_pool, dummy_pool, plan.info, plan.plan_dev, table, stable, q, 0.1,
                                            out, lse)
    assert e.value.status == 3
