"""GPU parity of the chunked branch prefill over the paged cache through the C ABI: chunks of query
tokens of branches (from their branch-initialization token or from the middle of the branch) and of
the prefix and layout stream, read from a paged bf16 pool in seeded random block order, against the
fp64 oracle's prefill rows of the same tokens of the packed pages (Sec. 3.2 visibility).

Tolerances as for the decode step: bf16 outputs max |d| <= 1.5e-2 and LSE <= 1e-3; fp32 1e-4.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import inputs
from paper_2608_06146_gb300 import padoc_attn as pa
from paper_2608_06146_gb300.engine import ChunkPrefillPlan
from paper_2608_06146_gb300.inputs import PageSpec, Workload

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _build():
    pbuild.build()
    pa.load_library()


def run_chunks(wl: Workload, seed: int, chunk_spec, scale_in=1.0, tc_ctas=0):
    """chunk_spec: list of (page, branch k or -1 for shared-stream tokens, first token, count)."""
    di = inputs.decode_inputs(wl, seed, scale=scale_in)
    # packed K/V of every page as [X | layout | Y_1 | ... | Y_N], from the logical cache
    ks, vs, bases, ybase = [], [], [], []
    base, b_idx = 0, 0
    for p, pg in enumerate(wl.pages):
        lo, n = int(di.page_off[p]), pg.stream_len
        ks.append(di.stream_k[lo:lo + n]); vs.append(di.stream_v[lo:lo + n])
        yb = []
        off = pg.stream_len
        for kb in range(pg.num_branches):
            plo, pn = int(di.priv_off[b_idx]), int(di.priv_len[b_idx])
            ks.append(di.priv_k[plo:plo + pn]); vs.append(di.priv_v[plo:plo + pn])
            yb.append(off)
            off += pn
            b_idx += 1
        bases.append(base)
        ybase.append(yb)
        base += pg.packed_len
    K, V = torch.cat(ks), torch.cat(vs)
    Q = inputs.randn((base, wl.num_q_heads, wl.head_dim), wl.dtype, seed * 1000 + 99, scale_in)
    chunks, table, rows = [], [], []
    first_branch = np.concatenate([[0], np.cumsum([pg.num_branches for pg in wl.pages])]).astype(int)
    for p, kb, a, n in chunk_spec:
        pg = wl.pages[p]
        if kb < 0:
            chunks.append((p, a, -1, n))
            table.append(np.full(di.stream_table.shape[1], -1, np.int32))
            rows += [bases[p] + a + i for i in range(n)]
        else:
            chunks.append((p, pg.prefix_len + pg.fork_offset[kb], a, n))
            table.append(di.stream_table[first_branch[p] + kb])
            rows += [bases[p] + ybase[p][kb] + a + i for i in range(n)]
    page_len = np.array([pg.stream_len for pg in wl.pages], np.int32)
    plan = ChunkPrefillPlan(page_len, chunks, np.stack(table), wl.num_q_heads, wl.num_kv_heads, wl.head_dim, DEV,
                            tc_ctas=tc_ctas)
    T = plan.num_tokens
    assert T == len(rows)
    q = Q[torch.as_tensor(rows)].contiguous().to(DEV)
    out = torch.full((T, wl.num_q_heads, wl.head_dim), float("nan"), dtype=wl.dtype, device=DEV)
    lse = torch.full((T, wl.num_q_heads), float("nan"), dtype=torch.float32, device=DEV)
    scale = 1.0 / math.sqrt(wl.head_dim)
    plan.run(di.k_pool.to(DEV), di.v_pool.to(DEV), torch.from_numpy(di.page_table).to(DEV), q, scale, out, lse)
    pa.padoc_check_device_errors()
    ref_o, ref_lse = oracle.prefill_dense(wl.pages, Q, K, V, scale)
    return out.float().cpu().numpy(), lse.cpu().numpy(), ref_o[rows], ref_lse[rows]


def assert_close(o, l, ro, rl, dtype):
    to, tl = (1.5e-2, 1e-3) if dtype == torch.bfloat16 else (1e-4, 1e-4)
    assert np.isfinite(o).all() and np.isfinite(l).all()
    do, dl = np.abs(o - ro).max(), np.abs(l - rl).max()
    assert do <= to, f"max |dO| = {do:.3e}"
    assert dl <= tl, f"max |dLSE| = {dl:.3e}"


PAGES = [PageSpec(700, 48, [48, 3, 20, 20, 0], [130, 9, 40, 1, 77]),
         PageSpec(90, 16, [16, 8], [33, 8]),
         PageSpec(2100, 200, [200, 150, 100], [260, 64, 31])]


def test_chunk_prefill_bf16_branch_and_shared_chunks():
    wl = Workload("chunk pages", PAGES, 16, 2, 128, torch.bfloat16, "decode")
    spec = [(0, 0, 0, 130), (0, 1, 0, 9), (0, 2, 7, 33), (0, 3, 0, 1), (0, 4, 40, 37), (0, -1, 700, 48),
            (0, -1, 0, 32), (1, 0, 0, 33), (1, 1, 1, 7), (1, -1, 90, 16),
            (2, 0, 0, 260), (2, 1, 0, 64), (2, 2, 0, 31), (2, -1, 2000, 300)]
    assert_close(*run_chunks(wl, 21, spec), torch.bfloat16)


@pytest.mark.parametrize("tc_ctas", [1, 5])
def test_chunk_prefill_bf16_few_ctas(tc_ctas):
    wl = Workload("chunk pages", PAGES, 16, 2, 128, torch.bfloat16, "decode")
    spec = [(0, 0, 30, 100), (0, 2, 0, 40), (2, 0, 0, 260), (2, -1, 1000, 200)]
    assert_close(*run_chunks(wl, 22, spec, tc_ctas=tc_ctas), torch.bfloat16)


def test_chunk_prefill_fp32_tiny():
    wl = inputs.tiny_page()
    pg = wl.pages[0]
    spec = [(0, k, 0, pg.branch_len[k]) for k in range(pg.num_branches)] + [(0, -1, 250, 38)]
    assert_close(*run_chunks(wl, 0, spec, scale_in=1 / 8), torch.float32)


def test_chunk_prefill_serving_batch_at_benchmark_size_sampled_rows():
    # the benchmarked branch prefill: the 32 serving-batch pages, every branch as one chunk from its
    # branch-initialization token and every layout stream as one shared-stream chunk (704 chunks,
    # 115,034 query tokens), in the launch configuration the benchmark times; the first, a middle
    # and the last token of every chunk (every page, every branch, every layout stream) against the
    # dense oracle's rows of those tokens of the packed pages
    wl = inputs.serving_batch(seed=3)
    di = inputs.decode_inputs(wl, 3, pool_slack=1.0)
    ks, vs, chunks, table, packed = [], [], [], [], []
    base, b = 0, 0
    for p, pg in enumerate(wl.pages):
        lo = int(di.page_off[p])
        ks.append(di.stream_k[lo:lo + pg.stream_len]); vs.append(di.stream_v[lo:lo + pg.stream_len])
        yb = base + pg.stream_len
        for f, n in zip(pg.fork_offset, pg.branch_len):
            plo = int(di.priv_off[b])
            ks.append(di.priv_k[plo:plo + n]); vs.append(di.priv_v[plo:plo + n])
            chunks.append((p, pg.prefix_len + f, 0, n))
            table.append(di.stream_table[b])
            packed.append(np.arange(yb, yb + n))
            yb += n
            b += 1
        chunks.append((p, pg.prefix_len, -1, pg.layout_len))
        table.append(np.full(di.stream_table.shape[1], -1, np.int32))
        packed.append(np.arange(base + pg.prefix_len, base + pg.stream_len))
        base += pg.packed_len
    K, V = torch.cat(ks), torch.cat(vs)
    page_len = np.array([pg.stream_len for pg in wl.pages], np.int32)
    plan = ChunkPrefillPlan(page_len, chunks, np.stack(table), 16, 2, 128, DEV)
    T = plan.num_tokens
    assert len(chunks) == 704 and T == 115034
    q = inputs.randn((T, 16, 128), torch.bfloat16, 3 * 1000 + 98)
    out = torch.full((T, 16, 128), float("nan"), dtype=torch.bfloat16, device=DEV)
    lse = torch.full((T, 16), float("nan"), dtype=torch.float32, device=DEV)
    scale = 1.0 / math.sqrt(128)
    plan.run(di.k_pool.to(DEV), di.v_pool.to(DEV), torch.from_numpy(di.page_table).to(DEV), q.to(DEV), scale, out, lse)
    pa.padoc_check_device_errors()
    tok, rows, t0 = [], [], 0
    for c, rr in zip(chunks, packed):
        n = c[3]
        for i in sorted({0, n // 2, n - 1}):
            tok.append(t0 + i)
            rows.append(int(rr[i]))
        t0 += n
    tok = np.array(tok)
    ref_o, ref_l = oracle.prefill_dense_rows(wl.pages, q[torch.from_numpy(tok)], K, V, scale, np.array(rows))
    got_o, got_l = out[torch.from_numpy(tok).to(DEV)].float().cpu().numpy(), lse[torch.from_numpy(tok).to(DEV)].cpu().numpy()
    assert_close(got_o, got_l, ref_o, ref_l, torch.bfloat16)
