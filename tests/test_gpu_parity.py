"""GPU parity: the CUDA path through the C ABI against the fp64 oracle, element by element, on the
same seeded inputs.

Tolerances: bf16 inputs with fp32 accumulation, outputs max |d| <= 1.5e-2 and LSE max |d| <= 1e-3;
the fp32 bring-up path (FMA in fp32, no tensor cores) <= 1e-4 for both.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import inputs
from paper_2608_06146_gb300 import padoc_attn as pa
from paper_2608_06146_gb300.engine import DecodePlan, PrefillPlan
from paper_2608_06146_gb300.inputs import PageSpec, Workload

pytestmark = pytest.mark.gpu

BF16_O_TOL, BF16_LSE_TOL = 1.5e-2, 1e-3
F32_TOL = 1e-4
DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _build():
    pbuild.build()
    pa.load_library()


def _tols(dtype):
    return (BF16_O_TOL, BF16_LSE_TOL) if dtype == torch.bfloat16 else (F32_TOL, F32_TOL)


def run_decode(wl: Workload, seed: int, layout_streams=False, split_tokens=0, scale_in=1.0, tc_ctas=0,
               warp_ctas=0):
    di = inputs.decode_inputs(wl, seed, layout_streams=layout_streams, scale=scale_in)
    plan = DecodePlan(wl.pages, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, DEV, wl.block_size, layout_streams,
                      split_tokens, tc_ctas, warp_ctas)
    S = plan.num_streams
    q = di.q.to(DEV)
    out = torch.full((S, wl.num_q_heads, wl.head_dim), float("nan"), dtype=wl.dtype, device=DEV)
    lse = torch.full((S, wl.num_q_heads), float("nan"), dtype=torch.float32, device=DEV)
    scale = 1.0 / math.sqrt(wl.head_dim)
    args = (di.k_pool.to(DEV), di.v_pool.to(DEV), torch.from_numpy(di.page_table).to(DEV),
            torch.from_numpy(di.stream_table).to(DEV), q, scale)
    plan.run(*args, out, lse)
    # a second call on the same plan and workspace gives a bit-identical result (every partial and
    # the merge's order are fixed by the plan)
    out2, lse2 = torch.full_like(out, float("nan")), torch.full_like(lse, float("nan"))
    plan.run(*args, out2, lse2)
    pa.padoc_check_device_errors()
    assert torch.equal(out, out2) and torch.equal(lse, lse2)
    ref_o, ref_lse = oracle.decode_pages(wl.pages, di, scale, layout_streams)
    return out.float().cpu().numpy(), lse.cpu().numpy(), ref_o, ref_lse


def assert_close(got_o, got_lse, ref_o, ref_lse, dtype):
    to, tl = _tols(dtype)
    assert np.isfinite(got_o).all() and np.isfinite(got_lse).all()
    do = np.abs(got_o - ref_o).max()
    dl = np.abs(got_lse - ref_lse).max()
    assert do <= to, f"max |dO| = {do:.3e} > {to}"
    assert dl <= tl, f"max |dLSE| = {dl:.3e} > {tl}"


# --------------------------------------------------------------------------------------------
# Decode
# --------------------------------------------------------------------------------------------

def test_decode_tiny_fp32():
    wl = inputs.tiny_page()
    assert_close(*run_decode(wl, 0, scale_in=1 / 8), torch.float32)


def test_decode_tiny_fp32_one_new_token_appended():
    wl = inputs.tiny_page()
    pg = wl.pages[0]
    wl.pages = [PageSpec(pg.prefix_len, pg.layout_len, pg.fork_offset, [n + 1 for n in pg.branch_len])]
    assert_close(*run_decode(wl, 5, layout_streams=True, scale_in=1 / 8), torch.float32)


@pytest.mark.parametrize("wl_name", ["decode_page", "dense_page", "serving_batch"])
def test_decode_bf16_workloads(wl_name):
    wl = inputs.WORKLOADS[wl_name]()
    assert_close(*run_decode(wl, 1), torch.bfloat16)


def test_decode_bf16_with_layout_streams_and_small_splits():
    wl = inputs.decode_page()
    assert_close(*run_decode(wl, 2, layout_streams=True, split_tokens=64), torch.bfloat16)


def test_decode_bf16_edge_pages():
    # f_k = 0 (prefix only), f_k = L, ties, a one-token branch, a page with P = 0 and unaligned
    # stream lengths, a page with a single branch, a long private history
    pages = [
        PageSpec(37, 9, [0, 9, 9, 4], [1, 17, 33, 2]),
        PageSpec(0, 5, [0, 5], [3, 1]),
        PageSpec(1000, 24, [24], [700]),
        PageSpec(16, 0, [0, 0, 0, 0, 0, 0], [16, 15, 14, 1, 2, 3]),
    ]
    wl = Workload("edge", pages, 16, 2, 128, torch.bfloat16, "decode")
    assert_close(*run_decode(wl, 3, layout_streams=True), torch.bfloat16)


def test_decode_bf16_tensor_core_edge_pages():
    # pages whose branches x heads fill M = 128 tiles: 10 branches (one M-tile), 17 (two M-tiles, the
    # second nearly empty), 33 (two items of 32 + 1 streams); unaligned shared lengths, f_k = 0 and
    # f_k = L ties, one-token private histories and a split boundary inside the layout stream
    rng = np.random.default_rng(8)
    def page(P, L, n):
        forks = [int(x) for x in rng.integers(0, L + 1, size=n)]
        forks[0], forks[-1] = 0, L
        lens = [int(x) for x in rng.integers(1, 300, size=n)]
        lens[1] = 1
        return PageSpec(P, L, forks, lens)
    pages = [page(37, 21, 10), page(700, 40, 17), page(1200, 264, 33), page(5, 3, 8)]
    wl = Workload("tc edge", pages, 16, 2, 128, torch.bfloat16, "decode")
    assert_close(*run_decode(wl, 9, layout_streams=True), torch.bfloat16)
    assert_close(*run_decode(wl, 10, split_tokens=128), torch.bfloat16)


@pytest.mark.parametrize("tc_ctas,warp_ctas", [(1, 1), (3, 2), (7, 5), (40, 0), (5, 400), (1000, 1000)])
def test_decode_bf16_tensor_core_ctas_walk_many_pieces(tc_ctas, warp_ctas):
    # few CTAs: each walks many pieces of different pages, KV heads and M-tile counts back to back
    # (the K/V ring, barrier phases and query reloads carry across pieces), and each warp of the
    # warp kernel walks a long list of items with one cp.async ring; many CTAs: one-tile pieces,
    # CTAs with empty ranges and one item per warp
    rng = np.random.default_rng(11)
    pages = []
    for n in [40, 9, 17, 33, 12, 64, 8]:
        P, L = int(rng.integers(1, 1500)), 8 * n
        pages.append(PageSpec(P, L, [int(x) for x in rng.integers(0, L + 1, size=n)],
                              [int(x) for x in rng.integers(1, 200, size=n)]))
    wl = Workload("tc walk", pages, 16, 2, 128, torch.bfloat16, "decode")
    assert_close(*run_decode(wl, 12, layout_streams=bool(tc_ctas & 1), tc_ctas=tc_ctas, warp_ctas=warp_ctas),
                 torch.bfloat16)


def test_decode_bf16_serving_batch_warp_ctas_beyond_the_sm_count():
    # few tensor-core CTAs and more warp CTAs than SMs: the grid holds more CTAs than fit at once,
    # so warp CTAs past the SM count start only as others end (the pairing of warp CTAs with
    # tensor-core CTAs in plan_internal.h)
    wl = inputs.serving_batch()
    assert_close(*run_decode(wl, 13, tc_ctas=5, warp_ctas=400), torch.bfloat16)


@pytest.mark.parametrize("prefix,split,merge", [(1000, 64, "wide"), (3000, 64, "cluster"), (4000, 0, "cluster")])
def test_decode_bf16_many_partials_per_key(prefix, split, merge):
    """Few streams with long shared streams cut into short items: every (stream, KV head) key has
    many partials, which the merge joins with four thread groups per key (9 to 32 partials) or a
    cluster of eight CTAs per key joined through distributed shared memory (more); split 0 is the
    planner's own choice for so little work (64-token items)."""
    pages = [PageSpec(prefix, 40, [0, 17, 40], [1500, 33, 260]), PageSpec(prefix // 2, 0, [0, 0], [700, 1])]
    wl = Workload("many partials", pages, 16, 2, 128, torch.bfloat16, "decode")
    plan = DecodePlan(wl.pages, 16, 2, 128, DEV, 16, False, split)
    info = plan.info
    assert info.num_merge_keys * 8 <= 2 * 152 and (32 < info.max_stream_slots if merge == "cluster" else
                                                   8 < info.max_stream_slots <= 32)
    assert_close(*run_decode(wl, 21, split_tokens=split), torch.bfloat16)


def test_decode_bf16_sparse_pages_on_tensor_cores():
    """Pages of two to seven streams whose plan has much warp work (few warp CTAs): their shared
    streams go to the tensor cores, one M-tile of 16 stream slots per group, mostly empty rows."""
    rng = np.random.default_rng(5)
    pages = []
    for n in (2, 3, 5, 7, 2):
        L = int(rng.integers(0, 60))
        pages.append(PageSpec(int(rng.integers(300, 1500)), L, [int(x) for x in rng.integers(0, L + 1, n)],
                              [int(x) for x in rng.integers(1, 400, n)]))
    wl = Workload("sparse pages", pages, 16, 2, 128, torch.bfloat16, "decode")
    plan = DecodePlan(wl.pages, 16, 2, 128, DEV, 16, False, 0, 0, 2)
    items = plan.plan_host[plan.info.off_items:plan.info.off_items + 8 * plan.info.num_tc_items].reshape(-1, 8)
    assert plan.info.num_tc_items > 0 and {0, 1, 4} <= set(int(i) for i in items[:, 1])
    assert_close(*run_decode(wl, 23, warp_ctas=2), torch.bfloat16)
    assert_close(*run_decode(wl, 24, layout_streams=True, warp_ctas=2), torch.bfloat16)


def test_decode_repeated_calls_on_one_workspace():
    # one plan and workspace serve several calls with new inputs; each call is exact
    wl = inputs.serving_batch(num_pages=6)
    plan = DecodePlan(wl.pages, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, DEV)
    for seed in (31, 32, 33):
        di = inputs.decode_inputs(wl, seed)
        S = plan.num_streams
        out = torch.full((S, 16, 128), float("nan"), dtype=torch.bfloat16, device=DEV)
        lse = torch.full((S, 16), float("nan"), dtype=torch.float32, device=DEV)
        scale = 1.0 / math.sqrt(wl.head_dim)
        plan.run(di.k_pool.to(DEV), di.v_pool.to(DEV), torch.from_numpy(di.page_table).to(DEV),
                 torch.from_numpy(di.stream_table).to(DEV), di.q.to(DEV), scale, out, lse)
        pa.padoc_check_device_errors()
        ref_o, ref_lse = oracle.decode_pages(wl.pages, di, scale)
        assert_close(out.float().cpu().numpy(), lse.cpu().numpy(), ref_o, ref_lse, torch.bfloat16)


def test_decode_bad_block_id_reports_device_error():
    wl = inputs.decode_page()
    di = inputs.decode_inputs(wl, 4)
    plan = DecodePlan(wl.pages, 16, 2, 128, DEV)
    table = di.page_table.copy()
    table[0, 3] = di.num_blocks + 5         # out of range: the kernel skips it and records the id
    S = plan.num_streams
    out = torch.empty((S, 16, 128), dtype=torch.bfloat16, device=DEV)
    lse = torch.empty((S, 16), dtype=torch.float32, device=DEV)
    plan.run(di.k_pool.to(DEV), di.v_pool.to(DEV), torch.from_numpy(table).to(DEV),
             torch.from_numpy(di.stream_table).to(DEV), di.q.to(DEV), 0.088, out, lse)
    with pytest.raises(pa.PadocError) as e:
        pa.padoc_check_device_errors()
    assert e.value.device_code == 1 and e.value.device_detail == di.num_blocks + 5
    pa.padoc_check_device_errors()          # the word was cleared


# --------------------------------------------------------------------------------------------
# Split-K combine (C4)
# --------------------------------------------------------------------------------------------

@pytest.mark.parametrize("S,R,d", [(1, 5, 128), (7, 300, 128), (3, 64, 64)])
def test_splitk_combine_matches_oracle_merge(S, R, d):
    g = torch.Generator().manual_seed(S * 100 + R)
    po = torch.randn(S, R, d, generator=g)
    pl = torch.randn(S, R, generator=g) * 4
    pl[0, : R // 3] = float("-inf")          # empty parts weigh nothing
    if S > 1:
        pl[:, :2] = float("-inf")            # rows with no visible key at all
    for dt in (torch.float32, torch.bfloat16):
        out = torch.empty(R, d, dtype=dt, device=DEV)
        lse = torch.empty(R, dtype=torch.float32, device=DEV)
        pa.padoc_splitk_combine(po.to(DEV), pl.to(DEV), out, lse)
        torch.cuda.synchronize()
        ref_o, ref_l = oracle.merge(po.double().numpy(), pl.double().numpy())
        got_l = lse.cpu().numpy()
        fin = np.isfinite(ref_l)
        np.testing.assert_array_equal(np.isneginf(got_l), ~fin)
        tol = 1e-5 if dt == torch.float32 else 1e-2
        assert np.abs(out.float().cpu().numpy() - ref_o).max() <= tol
        assert np.abs(got_l[fin] - ref_l[fin]).max() <= 1e-5


# --------------------------------------------------------------------------------------------
# Prefill
# --------------------------------------------------------------------------------------------

def run_prefill(wl: Workload, seed: int, scale_in=1.0, ref="gather"):
    q, k, v = inputs.packed_qkv(wl, seed, scale_in)
    plan = PrefillPlan(wl.pages, wl.dtype, wl.head_dim, DEV)
    T = plan.T
    out = torch.full((T, wl.num_q_heads, wl.head_dim), float("nan"), dtype=wl.dtype, device=DEV)
    lse = torch.full((T, wl.num_q_heads), float("nan"), dtype=torch.float32, device=DEV)
    scale = 1.0 / math.sqrt(wl.head_dim)
    plan.run(q.to(DEV), k.to(DEV), v.to(DEV), scale, out, lse)
    pa.padoc_check_device_errors()
    fn = oracle.prefill_gather if ref == "gather" else oracle.prefill_dense
    ref_o, ref_lse = fn(wl.pages, q, k, v, scale)
    return out.float().cpu().numpy(), lse.cpu().numpy(), ref_o, ref_lse


def test_prefill_tiny_fp32():
    wl = inputs.tiny_page()
    assert_close(*run_prefill(wl, 0, scale_in=1 / 8, ref="dense"), torch.float32)


def test_prefill_bf16_multi_page_ragged():
    # several 128-row tiles per page, pages not aligned to tiles, a ragged last tile, shuffled forks
    pages = [PageSpec(300, 40, [8, 40, 16, 0, 24], [50, 1, 77, 130, 9]),
             PageSpec(129, 0, [0, 0], [3, 200]),
             PageSpec(5, 16, [16], [1]),
             PageSpec(257, 64, [], [])]
    wl = Workload("ragged", pages, 16, 2, 128, torch.bfloat16, "prefill")
    assert_close(*run_prefill(wl, 6), torch.bfloat16)


def test_prefill_bf16_gqa_other_group_sizes():
    pages = [PageSpec(200, 16, [8, 16, 4], [40, 30, 60])]
    for hq, hkv in [(8, 8), (4, 1), (6, 2)]:
        wl = Workload("gqa", pages, hq, hkv, 128, torch.bfloat16, "prefill")
        assert_close(*run_prefill(wl, 7), torch.bfloat16)


def test_prefill_bf16_packed_full_size():
    # 8 pages x 4096 tokens, every row of every page against the oracle
    wl = inputs.packed_prefill()
    assert_close(*run_prefill(wl, 4), torch.bfloat16)


def test_prefill_bf16_packed_shuffled_branches_two_pages():
    wl = inputs.packed_prefill(seed=5, num_pages=2, shuffle_branches=True)
    assert_close(*run_prefill(wl, 5), torch.bfloat16)
