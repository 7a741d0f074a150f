"""GPU parity of the FP8 (E4M3) KV cache: quantization and append against the oracle bit for bit
(integer / byte work), and the decode step against the oracle's decode over the dequantized values
of the very codes the GPU holds, element by element.

Tolerance of the decode (outputs max |d| <= 1.5e-2, LSE max |d| <= 1e-3, those of the bf16 path):
the oracle attends over code_value * scale exactly (fp64), and so does the kernel up to its own
arithmetic. Codes become bf16 exactly (value x 2^-112, every E4M3 value has 4 significant bits),
the K scale multiplies each block's fp32 scores, and the V scale multiplies each fp32 probability
before the same bf16 rounding of P the bf16 path makes (relative 2^-9), while the row sum keeps the
unrounded probabilities. The remaining error sources (fp32 accumulation, ex2.approx, P in bf16) are
those of the bf16 path, on values of the same size (a block's largest magnitude is its bf16 one),
so its tolerances apply unchanged.
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
from paper_2608_06146_gb300.inputs import PageSpec, Workload

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
O_TOL, LSE_TOL = 1.5e-2, 1e-3


@pytest.fixture(scope="module", autouse=True)
def _build():
    pbuild.build()
    pa.load_library()


def _codes(pool):
    return (pool.k_codes.cpu().numpy(), pool.k_scales.cpu().numpy(), pool.v_codes.cpu().numpy(),
            pool.v_scales.cpu().numpy())


def quantized_inputs(wl, seed, layout_streams=False):
    di = inputs.decode_inputs(wl, seed, layout_streams=layout_streams)
    pool = pa.E4M3Pool(di.num_blocks, wl.num_kv_heads, wl.head_dim, DEV)
    blocks = torch.arange(di.num_blocks, dtype=torch.int32, device=DEV)
    pa.padoc_quantize_kv_blocks(pool, di.k_pool.to(DEV), di.v_pool.to(DEV), blocks)
    pa.padoc_check_device_errors()
    return di, pool


def run_decode_e4m3(wl, seed, layout_streams=False, split_tokens=0, tc_ctas=0, warp_ctas=0, di_pool=None):
    di, pool = di_pool or quantized_inputs(wl, seed, layout_streams)
    plan = DecodePlan(wl.pages, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, DEV, 16, layout_streams, split_tokens,
                      tc_ctas, warp_ctas)
    S = plan.num_streams
    out = torch.full((S, wl.num_q_heads, wl.head_dim), float("nan"), dtype=torch.bfloat16, device=DEV)
    lse = torch.full((S, wl.num_q_heads), float("nan"), dtype=torch.float32, device=DEV)
    scale = 1.0 / math.sqrt(wl.head_dim)
    pt, st, q = torch.from_numpy(di.page_table).to(DEV), torch.from_numpy(di.stream_table).to(DEV), di.q.to(DEV)
    pa.padoc_branch_decode_attn_e4m3(pool, plan.info, plan.plan_dev, pt, st, q, scale, out, lse, plan.workspace)
    # a second call on the same plan and workspace: bit-identical
    out2, lse2 = torch.full_like(out, float("nan")), torch.full_like(lse, float("nan"))
    pa.padoc_branch_decode_attn_e4m3(pool, plan.info, plan.plan_dev, pt, st, q, scale, out2, lse2, plan.workspace)
    pa.padoc_check_device_errors()
    assert torch.equal(out, out2) and torch.equal(lse, lse2)
    kc, ks, vc, vs = _codes(pool)
    ref_o, ref_l = oracle.decode_paged(wl.pages, oracle.dequantize_kv_blocks(kc, ks), oracle.dequantize_kv_blocks(vc, vs),
                                       di.page_table, di.stream_table, di.q, scale, layout_streams)
    got_o, got_l = out.float().cpu().numpy(), lse.cpu().numpy()
    assert np.isfinite(got_o).all() and np.isfinite(got_l).all()
    do, dl = np.abs(got_o - ref_o).max(), np.abs(got_l - ref_l).max()
    assert do <= O_TOL, f"max |dO| = {do:.3e}"
    assert dl <= LSE_TOL, f"max |dLSE| = {dl:.3e}"
    return plan


# ------------------------------------------------------------------------------------------------
# Quantization and append: bit-exact
# ------------------------------------------------------------------------------------------------

def test_quantize_blocks_bit_exact_against_oracle():
    wl = inputs.decode_page()
    di, pool = quantized_inputs(wl, 51)            # partly filled and unused (all-zero) blocks included
    kc, ks, vc, vs = _codes(pool)
    want_kc, want_ks = oracle.quantize_kv_blocks(di.k_pool)
    want_vc, want_vs = oracle.quantize_kv_blocks(di.v_pool)
    np.testing.assert_array_equal(ks, want_ks)
    np.testing.assert_array_equal(vs, want_vs)
    np.testing.assert_array_equal(kc, want_kc)
    np.testing.assert_array_equal(vc, want_vc)
    assert (ks == 0).any() and (ks > 0).any()


def test_quantize_ties_saturation_and_subnormals_bit_exact():
    # blocks whose largest magnitude is 448 have scale 1 exactly, so x / scale = x: every midpoint
    # between neighbouring codes (a tie, rounded to the even code), every code value, subnormal
    # values and signed zeros go through the kernel's conversion as they are
    vals = oracle.e4m3_decode(np.arange(0, 0x7F, dtype=np.uint8))
    mids = (vals[:-1] + vals[1:]) / 2
    x = np.concatenate([vals, mids, -vals, -mids, [2.0 ** -10, 3 * 2.0 ** -10, -0.0]])
    n = 4 * 16 * 128
    x = np.resize(x, n).astype(np.float32)
    rng = np.random.default_rng(7)
    x = rng.permutation(x).reshape(4, 1, 16, 128)
    x[:, 0, 0, 0] = 448.0
    src = torch.from_numpy(x).to(torch.bfloat16)
    assert torch.equal(src.float(), torch.from_numpy(x))   # bf16 holds them exactly
    pool = pa.E4M3Pool(4, 1, 128, DEV)
    pa.padoc_quantize_kv_blocks(pool, src.to(DEV), src.to(DEV), torch.arange(4, dtype=torch.int32, device=DEV))
    pa.padoc_check_device_errors()
    kc, ks, vc, vs = _codes(pool)
    want_c, want_s = oracle.quantize_kv_blocks(x)
    np.testing.assert_array_equal(ks, want_s)
    assert (ks == 1.0).all()
    np.testing.assert_array_equal(kc, want_c)
    np.testing.assert_array_equal(vc, want_c)


def test_append_rows_bit_exact_against_oracle_rule():
    # 12 blocks filled over 20 steps; each step appends one row to each of a subset of the blocks
    # (distinct blocks within a call), rows in order inside a block; magnitudes grow and shrink so
    # that scales grow (re-encoding earlier rows) and stay; every block starts with stale codes and
    # scales from a former owner and is started afresh at row 0; a zero row and a block of zero rows
    rng = np.random.default_rng(12)
    nb, hkv, d = 12, 2, 128
    kc0 = rng.integers(0, 0x7E, (nb, hkv, 16, d)).astype(np.uint8)
    vc0 = rng.integers(0, 0x7E, (nb, hkv, 16, d)).astype(np.uint8)
    ks0 = rng.uniform(0.1, 2, (nb, hkv)).astype(np.float32)
    vs0 = rng.uniform(0.1, 2, (nb, hkv)).astype(np.float32)
    pool = pa.E4M3Pool(nb, hkv, d, DEV)
    pool.k_codes.copy_(torch.from_numpy(kc0)); pool.v_codes.copy_(torch.from_numpy(vc0))
    pool.k_scales.copy_(torch.from_numpy(ks0)); pool.v_scales.copy_(torch.from_numpy(vs0))
    want = [kc0.copy(), ks0.copy(), vc0.copy(), vs0.copy()]
    fill = np.zeros(nb, np.int64)
    for step in range(20):
        blocks = [b for b in range(nb) if fill[b] < 16 and rng.random() < 0.8]
        if not blocks:
            continue
        slots = np.array([b * 16 + fill[b] for b in blocks], np.int32)
        mag = np.exp(rng.uniform(-3, 3, (len(blocks), hkv, 1)))
        k = (rng.standard_normal((len(blocks), hkv, d)) * mag).astype(np.float32)
        v = (rng.standard_normal((len(blocks), hkv, d)) * mag[:, ::-1]).astype(np.float32)
        for i, b in enumerate(blocks):
            if b == 11 or (b == 10 and fill[b] == 2):
                k[i] = 0.0; v[i] = 0.0
        kb, vb = torch.from_numpy(k).to(torch.bfloat16), torch.from_numpy(v).to(torch.bfloat16)
        pa.padoc_append_inputs_e4m3(pool, kb.to(DEV), vb.to(DEV), torch.from_numpy(slots).to(DEV))
        want[0], want[1] = oracle.append_kv_quantized(want[0], want[1], slots, kb.float())
        want[2], want[3] = oracle.append_kv_quantized(want[2], want[3], slots, vb.float())
        for b in blocks:
            fill[b] += 1
    pa.padoc_check_device_errors()
    kc, ks, vc, vs = _codes(pool)
    np.testing.assert_array_equal(ks, want[1])
    np.testing.assert_array_equal(vs, want[3])
    np.testing.assert_array_equal(kc, want[0])
    np.testing.assert_array_equal(vc, want[2])
    assert (fill > 1).all() and ks[11].max() == 0.0


def test_append_copies_queries_in_call_order():
    rng = np.random.default_rng(13)
    pool = pa.E4M3Pool(4, 2, 128, DEV)
    src_k = torch.randn(9, 2, 128).to(torch.bfloat16).to(DEV)
    src_q = torch.randn(9, 16, 128).to(torch.bfloat16).to(DEV)
    rows = torch.tensor([7, 2, 5], dtype=torch.int32, device=DEV)
    slots = torch.tensor([0, 16, 35], dtype=torch.int32, device=DEV)
    q_dst = torch.zeros(3, 16, 128, dtype=torch.bfloat16, device=DEV)
    pa.padoc_append_inputs_e4m3(pool, src_k, src_k, slots, q_src=src_q, q_dst=q_dst, src_rows=rows)
    pa.padoc_check_device_errors()
    assert torch.equal(q_dst, src_q[rows.long()])


# ------------------------------------------------------------------------------------------------
# Decode over the E4M3 pool
# ------------------------------------------------------------------------------------------------

@pytest.mark.parametrize("wl_name", ["decode_page", "dense_page", "serving_batch"])
def test_decode_e4m3_workloads(wl_name):
    wl = inputs.WORKLOADS[wl_name]()
    plan = run_decode_e4m3(wl, 61)
    if wl_name != "decode_page":
        assert plan.info.num_tc_items > 0 and plan.info.num_warps > 0   # both kernels ran


def test_decode_e4m3_edge_pages_and_layout_streams():
    pages = [PageSpec(37, 9, [0, 9, 9, 4], [1, 17, 33, 2]), PageSpec(0, 5, [0, 5], [3, 1]),
             PageSpec(1000, 24, [24], [700]), PageSpec(16, 0, [0, 0, 0, 0, 0, 0], [16, 15, 14, 1, 2, 3])]
    wl = Workload("edge", pages, 16, 2, 128, torch.bfloat16, "decode")
    run_decode_e4m3(wl, 62, layout_streams=True)
    run_decode_e4m3(wl, 63, split_tokens=64)


@pytest.mark.parametrize("tc_ctas,warp_ctas", [(1, 1), (3, 2), (7, 5), (1000, 1000)])
def test_decode_e4m3_tensor_core_ctas_walk_many_pieces(tc_ctas, warp_ctas):
    # few CTAs: each walks pieces of different pages, KV heads and M-tile counts back to back, with
    # the expansion lagging the loads across piece boundaries; many CTAs: one-tile pieces
    rng = np.random.default_rng(11)
    pages = []
    for n in [40, 9, 17, 33, 12, 64, 8]:
        P, L = int(rng.integers(1, 1500)), 8 * n
        pages.append(PageSpec(P, L, [int(x) for x in rng.integers(0, L + 1, size=n)],
                              [int(x) for x in rng.integers(1, 200, size=n)]))
    wl = Workload("tc walk", pages, 16, 2, 128, torch.bfloat16, "decode")
    run_decode_e4m3(wl, 64, layout_streams=bool(tc_ctas & 1), tc_ctas=tc_ctas, warp_ctas=warp_ctas)


def test_decode_e4m3_scales_that_differ_block_by_block():
    # every block of the cache gets its own magnitude, so scales differ block by block (K over e^-3
    # .. e^1, V over e^-3 .. 1, independently), and some K blocks are all zero (scale 0): the per-
    # block K multipliers and V factors must follow. Magnitudes stay at most those of the N(0,1)
    # workloads' (|V| up to ~4.5) so that the bf16 path's absolute tolerances still apply: the
    # outputs' own bf16 rounding grows with |V|.
    wl = inputs.dense_page()
    di = inputs.decode_inputs(wl, 65)
    rng = np.random.default_rng(65)
    kmag = torch.from_numpy(np.exp(rng.uniform(-3, 1, (di.num_blocks, 2, 1, 1))).astype(np.float32))
    vmag = torch.from_numpy(np.exp(rng.uniform(-3, 0, (di.num_blocks, 2, 1, 1))).astype(np.float32))
    zero = torch.from_numpy(rng.random((di.num_blocks, 2, 1, 1)) < 0.05)
    di.k_pool = (di.k_pool.float() * kmag).masked_fill(zero, 0.0).to(torch.bfloat16)
    di.v_pool = (di.v_pool.float() * vmag).to(torch.bfloat16)
    pool = pa.E4M3Pool(di.num_blocks, 2, 128, DEV)
    pa.padoc_quantize_kv_blocks(pool, di.k_pool.to(DEV), di.v_pool.to(DEV),
                                torch.arange(di.num_blocks, dtype=torch.int32, device=DEV))
    run_decode_e4m3(wl, 65, di_pool=(di, pool))


def test_decode_e4m3_after_appends_matches_oracle():
    # a decoding loop's cache: the prefix quantized as whole blocks, then every branch's rows and the
    # layout stream's tail appended row by row (one row per stream per step, as Algorithm 1 does);
    # the decode of every stream's newest token against the oracle on the resulting codes
    pages = [PageSpec(300, 40, [8, 40, 16, 0, 24, 33], [50, 1, 77, 130, 9, 40]),
             PageSpec(129, 16, [0, 16, 3, 3, 12, 7, 1, 9, 16, 2], [3, 20, 33, 1, 17, 64, 5, 8, 2, 40])]
    wl = Workload("loop", pages, 16, 2, 128, torch.bfloat16, "decode")
    di = inputs.decode_inputs(wl, 66, layout_streams=True)
    pool = pa.E4M3Pool(di.num_blocks, 2, 128, DEV)
    # prefix blocks (all rows < P) whole; every other row of the cache appended row by row
    k_rows, v_rows, slots, order = [], [], [], []
    prefix_blocks = []
    for p, pg in enumerate(pages):
        nfull = pg.prefix_len // 16
        prefix_blocks += [int(b) for b in di.page_table[p, :nfull]]
        for t in range(nfull * 16, pg.stream_len):
            b = int(di.page_table[p, t // 16])
            k_rows.append(di.k_pool[b, :, t % 16]); v_rows.append(di.v_pool[b, :, t % 16])
            slots.append(b * 16 + t % 16); order.append(t % 16)
    for s in range(len(di.stream_page)):
        for t in range(int(di.priv_len[s])):
            b = int(di.stream_table[s, t // 16])
            k_rows.append(di.k_pool[b, :, t % 16]); v_rows.append(di.v_pool[b, :, t % 16])
            slots.append(b * 16 + t % 16); order.append(t % 16)
    blocks = torch.tensor(prefix_blocks, dtype=torch.int32, device=DEV)
    pa.padoc_quantize_kv_blocks(pool, di.k_pool[prefix_blocks].to(DEV), di.v_pool[prefix_blocks].to(DEV), blocks)
    k_rows, v_rows = torch.stack(k_rows), torch.stack(v_rows)
    slots, order = np.array(slots, np.int32), np.array(order)
    for r in range(16):   # step r appends row r of every block (distinct blocks within a call)
        idx = np.nonzero(order == r)[0]
        if len(idx):
            it = torch.from_numpy(idx)
            pa.padoc_append_inputs_e4m3(pool, k_rows[it].to(DEV), v_rows[it].to(DEV),
                                        torch.from_numpy(slots[idx]).to(DEV))
    pa.padoc_check_device_errors()
    run_decode_e4m3(wl, 66, layout_streams=True, di_pool=(di, pool))
