"""The host-side conveniences of a decode loop on the GPU: a plan advanced in place for longer
private histories decodes exactly what a plan built for those lengths would (checked against the
oracle), and the one-call step (copies in, decode, copies out) returns the oracle's results in host
memory. Tolerances of the bf16 decode: outputs 1.5e-2, LSE 1e-3."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import inputs
from paper_2608_06146_gb300 import padoc_attn as pa
from paper_2608_06146_gb300.inputs import PageSpec, Workload

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _build():
    pbuild.build()
    pa.load_library()


def _check(got_o, got_l, ref_o, ref_l):
    assert np.isfinite(got_o).all() and np.isfinite(got_l).all()
    assert np.abs(got_o - ref_o).max() <= 1.5e-2
    assert np.abs(got_l - ref_l).max() <= 1e-3


def test_advanced_plan_decodes_the_grown_batch():
    wl = inputs.serving_batch(num_pages=6, seed=5)
    rng = np.random.default_rng(5)
    grown = []
    for pg in wl.pages:   # 1 .. 60 more private rows per branch
        grown.append(PageSpec(pg.prefix_len, pg.layout_len, pg.fork_offset,
                              [n + int(rng.integers(1, 61)) for n in pg.branch_len]))
    cfg = pa.make_decode_config(16, 2, 128, 16, True, 0, 0, 0)
    plan, info = pa.padoc_build_decode_plan(wl.pages, cfg)
    plan = plan.copy()
    _, _, new_len = oracle.decode_streams(grown, True)
    assert pa.padoc_advance_decode_plan(plan, info, new_len)
    wl2 = Workload("grown", grown, 16, 2, 128, torch.bfloat16, "decode")
    di = inputs.decode_inputs(wl2, 5, layout_streams=True)
    S = info.num_streams
    out = torch.full((S, 16, 128), float("nan"), dtype=torch.bfloat16, device=DEV)
    lse = torch.full((S, 16), float("nan"), dtype=torch.float32, device=DEV)
    ws = torch.empty(pa.padoc_decode_workspace_size(info), dtype=torch.uint8, device=DEV)
    scale = 1.0 / math.sqrt(128)
    pa.padoc_branch_decode_attn(di.k_pool.to(DEV), di.v_pool.to(DEV), info, torch.from_numpy(plan).to(DEV),
                                torch.from_numpy(di.page_table).to(DEV), torch.from_numpy(di.stream_table).to(DEV),
                                di.q.to(DEV), scale, out, lse, ws)
    pa.padoc_check_device_errors()
    ref_o, ref_l = oracle.decode_pages(grown, di, scale, layout_streams=True)
    _check(out.float().cpu().numpy(), lse.cpu().numpy(), ref_o, ref_l)


@pytest.mark.parametrize("piped,prepared", [(False, False), (True, False), (True, True)])
def test_one_call_step_from_host_memory(piped, prepared):
    """padoc_launch_decode_step from pinned host memory, with the copies on the compute stream or on
    copy streams ordered by the buffer set's events; prepared: through pa.DecodeStep (arguments
    marshalled once; its plan advance to the same lengths changes nothing), three calls in a row."""
    wl = inputs.dense_page()
    di = inputs.decode_inputs(wl, 71)
    cfg = pa.make_decode_config(16, 2, 128, 16, False, 0, 0, 0)
    plan, info = pa.padoc_build_decode_plan(wl.pages, cfg)
    S = info.num_streams
    PT, STW = di.page_table.shape[1], di.stream_table.shape[1]
    a = lambda n: (n + 31) // 32 * 32
    off_pt = a(int(info.plan_ints))
    off_st = off_pt + a(PT)
    words = off_st + a(S * STW)
    stage = torch.zeros(words, dtype=torch.int32).pin_memory()
    h = stage.numpy()
    h[:info.plan_ints] = plan
    h[off_pt:off_pt + PT] = di.page_table.reshape(-1)
    h[off_st:off_st + S * STW] = di.stream_table.reshape(-1)
    dev_ints = torch.empty(words + 64, dtype=torch.int32, device=DEV)
    q_host = di.q.pin_memory()
    q_dev = torch.empty((S, 16, 128), dtype=torch.bfloat16, device=DEV)
    out = torch.empty_like(q_dev)
    lse = torch.empty((S, 16), dtype=torch.float32, device=DEV)
    o_host = torch.full((S, 16, 128), float("nan"), dtype=torch.bfloat16).pin_memory()
    l_host = torch.full((S, 16), float("nan"), dtype=torch.float32).pin_memory()
    ws = torch.empty(pa.padoc_decode_workspace_size(info), dtype=torch.uint8, device=DEV)
    scale = 1.0 / math.sqrt(128)
    kw = {}
    if piped:   # copies on their own streams, ordered by the buffer set's events
        evs = [torch.cuda.Event() for _ in range(3)]
        for e in evs:
            e.record()
        kw = dict(copy_in=torch.cuda.Stream(), copy_out=torch.cuda.Stream(), ev_free=evs[0], ev_in=evs[1], ev_dec=evs[2])
    k_pool, v_pool = di.k_pool.to(DEV), di.v_pool.to(DEV)
    if prepared:
        lens = plan[info.off_private_len:info.off_private_len + S].copy()
        step = pa.DecodeStep(k_pool, v_pool, info, stage, words, int(info.plan_ints), off_pt, PT, off_st, STW, dev_ints,
                             q_host, q_dev, scale, out, lse, o_host, l_host, ws, lens, **kw)
        for _ in range(3):
            kw["ev_in"].synchronize()       # the set's previous copies in have run
            assert step()
        np.testing.assert_array_equal(h[:info.plan_ints], plan)
    else:
        pa.padoc_launch_decode_step(k_pool, v_pool, info, stage, words, off_pt, PT, off_st, STW, dev_ints, q_host, q_dev,
                                    scale, out, lse, o_host, l_host, ws, **kw)
    if piped:
        kw["ev_free"].synchronize()         # the results' copies out have run
    pa.padoc_check_device_errors()          # synchronizes the stream: the results are in host memory
    ref_o, ref_l = oracle.decode_pages(wl.pages, di, scale)
    _check(o_host.float().numpy(), l_host.numpy(), ref_o, ref_l)
