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

import oracle
from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import inputs
from paper_2608_06146_gb300 import padoc_attn as pa
from paper_2608_06146_gb300.engine import DecodePlan

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
O_TOL, LSE_TOL = 1.5e-2, 1e-3   # the bf16 decode tolerances of the parity tests


def test_noalloc_decode_matches_oracle_and_workspace_decode_on_two_calls():
    pbuild.build()
    pa.load_library()
    wl = inputs.dense_page()                      # 64 branches on one page
    plan = DecodePlan(wl.pages, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, DEV)
    assert pa.padoc_decode_workspace_size(plan.info) <= pa.PADOC_STATIC_WORKSPACE_BYTES
    S = plan.num_streams
    scale = 1.0 / math.sqrt(wl.head_dim)
    for call, seed in enumerate((21, 22)):        # two calls in a row on different caches and queries
        di = inputs.decode_inputs(wl, seed)
        k_pool, v_pool = di.k_pool.to(DEV), di.v_pool.to(DEV)
        pt, st = torch.from_numpy(di.page_table).to(DEV), torch.from_numpy(di.stream_table).to(DEV)
        q = di.q.to(DEV)
        out = torch.full((S, 16, 128), float("nan"), dtype=torch.bfloat16, device=DEV)
        lse = torch.full((S, 16), float("nan"), dtype=torch.float32, device=DEV)
        pa.padoc_branch_decode_attn_noalloc(k_pool, v_pool, plan.info, plan.plan_dev, pt, st, q, scale, out, lse)
        pa.padoc_check_device_errors()
        got_o, got_l = out.float().cpu().numpy(), lse.cpu().numpy()
        assert np.isfinite(got_o).all() and np.isfinite(got_l).all(), f"call {call}: non-finite output"
        # against the fp64 oracle on the same inputs
        ref_o, ref_l = oracle.decode_pages(wl.pages, di, scale)
        do, dl = np.abs(got_o - ref_o).max(), np.abs(got_l - ref_l).max()
        assert do <= O_TOL, f"call {call}: max |dO| vs oracle = {do}"
        assert dl <= LSE_TOL, f"call {call}: max |dLSE| vs oracle = {dl}"
        # and against the entry point that takes a caller's workspace
        ws_o = torch.empty((S, 16, 128), dtype=torch.bfloat16, device=DEV)
        ws_l = torch.empty((S, 16), dtype=torch.float32, device=DEV)
        plan.run(k_pool, v_pool, pt, st, q, scale, ws_o, ws_l)
        pa.padoc_check_device_errors()
        do = (out.float() - ws_o.float()).abs().max().item()
        dl = (lse - ws_l).abs().max().item()
        assert do <= O_TOL, f"call {call}: max |dO| vs workspace decode = {do}"
        assert dl <= LSE_TOL, f"call {call}: max |dLSE| vs workspace decode = {dl}"


def test_noalloc_rejects_a_plan_beyond_the_array():
    pa.load_library()
    wl = inputs.serving_batch(num_pages=256)      # its split-K partials need more than 32 MiB
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
