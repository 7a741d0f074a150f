"""GPU parity of Algorithm 1's loop (App. E.1) through the C ABI: the scheduler (padoc_mpd_*),
the append kernel and the decode step run every page from its prefill to its last branch's EOS,
and every token the loop decodes must equal, within the decode tolerances, the fp64 oracle's
output for that token of the packed pages (the decode of a stream's newest token is the prefill
row of that token; the oracle pins that identity).

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
from paper_2608_06146_gb300.engine import MaskedParallelLoop
from paper_2608_06146_gb300.inputs import LoopTokenSource, PageSpec, Workload

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
BF16_O_TOL, BF16_LSE_TOL = 1.5e-2, 1e-3
F32_TOL = 1e-4


@pytest.fixture(scope="module", autouse=True)
def _build():
    pbuild.build()
    pa.load_library()


def _blocks_needed(pages, bs=16):
    return sum(-(-(pg.prefix_len + pg.layout_len) // bs) + sum(-(-n // bs) for n in pg.branch_len) for pg in pages)


def run_loop(wl: Workload, seed: int, admit_at=None, keep_rows=None, scale_in=1.0, slack=3, runner=False):
    """Runs the loop over wl.pages; returns (packed rows decoded, O fp32, LSE) of the kept rows
    (all rows when keep_rows is None) and the loop. runner: each step through the one-call runner
    (padoc_mpd_runner_step, source rows from a table by stream id) instead of prepare + launch."""
    q, k, v = inputs.packed_qkv(wl, seed, scale_in)
    qd, kd, vd = q.to(DEV), k.to(DEV), v.to(DEV)
    src = LoopTokenSource(wl.pages)
    nb = _blocks_needed(wl.pages) + slack
    order = np.random.default_rng(seed + 77).permutation(nb).astype(np.int32)
    loop = MaskedParallelLoop(nb, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.dtype, DEV, block_order=order)
    scale = 1.0 / math.sqrt(wl.head_dim)
    admit_at = admit_at or [0] * len(wl.pages)
    pending = sorted(range(len(wl.pages)), key=lambda p: admit_at[p])
    keep = None if keep_rows is None else set(int(r) for r in keep_rows)
    rows_out, o_out, l_out = [], [], []
    cap = sum(1 + pg.num_branches for pg in wl.pages)   # every stream id the loop can create
    out_buf = torch.empty((cap, wl.num_q_heads, wl.head_dim), dtype=wl.dtype, device=DEV)
    lse_buf = torch.empty((cap, wl.num_q_heads), dtype=torch.float32, device=DEV)
    row_of = np.zeros(cap, np.int32)
    step = 0
    while True:
        while pending and admit_at[pending[0]] <= step:
            p = pending.pop(0)
            P, nf, leos, prow = src.admission(p)
            _, new = loop.add_page(P, nf, leos, kd, vd, prow)
            src.admitted(p, new)
        if loop.status()[1] == 0:
            if not pending:
                break
            step += 1
            continue
        if runner:
            row_of[:] = src.peek_rows(np.arange(cap))
            n, ids = loop.run_step(kd, vd, qd, row_of, scale, out_buf, lse_buf)
            ids = ids.copy()
            assert np.array_equal(src.rows(ids), row_of[ids])
            out, lse = out_buf[:n], lse_buf[:n]
        else:
            ids, out, lse = loop.step(kd, vd, qd, src.rows, scale)
        rows = src.token_rows(ids)
        sel = np.arange(len(ids)) if keep is None else np.array([i for i, r in enumerate(rows) if int(r) in keep],
                                                                np.int64)
        if len(sel):
            idx = torch.from_numpy(sel).to(DEV)
            rows_out.append(rows[sel])
            o_out.append(out.index_select(0, idx).float())
            l_out.append(lse.index_select(0, idx))
        nf, eos = src.events(ids)
        src.forked(ids, nf, loop.end_step(nf, eos))
        step += 1
    pa.padoc_check_device_errors()
    assert loop.status() == (0, 0, nb), "every block returns to the pool"
    return (np.concatenate(rows_out), torch.cat(o_out).cpu().numpy(), torch.cat(l_out).cpu().numpy(), q, k, v,
            loop)


def assert_close(got_o, got_lse, ref_o, ref_lse, dtype):
    to, tl = (BF16_O_TOL, BF16_LSE_TOL) if dtype == torch.bfloat16 else (F32_TOL, F32_TOL)
    assert np.isfinite(got_o).all() and np.isfinite(got_lse).all()
    do = np.abs(got_o - ref_o).max()
    dl = np.abs(got_lse - ref_lse).max()
    assert do <= to, f"max |dO| = {do:.3e} > {to}"
    assert dl <= tl, f"max |dLSE| = {dl:.3e} > {tl}"


def check_all_rows(wl, seed, **kw):
    rows, o, lse, q, k, v, _ = run_loop(wl, seed, **kw)
    src = LoopTokenSource(wl.pages)
    want = sorted(int(src.base[p]) + j for p, pg in enumerate(wl.pages) for j in range(pg.prefix_len, pg.packed_len))
    assert sorted(rows.tolist()) == want, "each layout and branch token is decoded exactly once"
    ref_o, ref_lse = oracle.prefill_dense(wl.pages, q, k, v, 1.0 / math.sqrt(wl.head_dim))
    assert_close(o, lse, ref_o[rows], ref_lse[rows], wl.dtype)


def test_loop_tiny_fp32():
    wl = inputs.tiny_page()
    check_all_rows(wl, 0, scale_in=1 / 8)


def test_loop_bf16_edge_pages_staggered():
    """Forks at the prefill (f = 0) and at the layout stream's last token, tied and unordered fork
    offsets, a page without a layout stream, a page without a prefix, branches crossing block
    boundaries, and a page with enough live streams for the tensor-core shared-stream kernel;
    pages admitted while others decode."""
    pages = [PageSpec(37, 10, [0, 10, 3, 3, 7], [17, 5, 33, 1, 16]),
             PageSpec(50, 0, [0, 0], [20, 3]),
             PageSpec(0, 6, [6, 2], [4, 18]),
             PageSpec(300, 40, [40, 4, 8, 12, 16, 20, 24, 28, 32, 36, 0, 1], [40, 35, 3, 60, 22, 17, 16, 33, 48, 9,
                                                                               12, 25]),
             PageSpec(130, 24, [24, 12], [2, 70])]
    wl = Workload("loop edge pages", pages, 16, 2, 128, torch.bfloat16, "decode")
    check_all_rows(wl, 5, admit_at=[0, 0, 4, 6, 30])


def test_loop_runner_matches_two_call_loop():
    """The one-call runner (padoc_mpd_runner_step) and the prepare + launch path make the same steps:
    the same streams in the same order and bit-identical outputs and LSE, on the edge pages with
    staggered admission; both match the oracle."""
    pages = [PageSpec(37, 10, [0, 10, 3, 3, 7], [17, 5, 33, 1, 16]),
             PageSpec(50, 0, [0, 0], [20, 3]),
             PageSpec(0, 6, [6, 2], [4, 18]),
             PageSpec(300, 40, [40, 4, 8, 12, 16, 20, 24, 28, 32, 36, 0, 1], [40, 35, 3, 60, 22, 17, 16, 33, 48, 9,
                                                                               12, 25])]
    wl = Workload("loop runner pages", pages, 16, 2, 128, torch.bfloat16, "decode")
    a = run_loop(wl, 6, admit_at=[0, 2, 5, 9])
    b = run_loop(wl, 6, admit_at=[0, 2, 5, 9], runner=True)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])
    np.testing.assert_array_equal(a[2], b[2])
    q, k, v = b[3], b[4], b[5]
    ref_o, ref_lse = oracle.prefill_dense(wl.pages, q, k, v, 1.0 / math.sqrt(wl.head_dim))
    assert_close(b[1], b[2], ref_o[b[0]], ref_lse[b[0]], wl.dtype)


def test_loop_bf16_serving_batch_sampled():
    """The 32-page serving batch (prefix 1024-4096, Poisson(20) branches, log-normal branch lengths)
    decoded from prefill to the last EOS; 400 decoded tokens, drawn at random, against the oracle's
    decode of that token's stream (its shared cutoff and private rows, the decode = prefill row
    identity)."""
    wl = inputs.serving_batch(seed=3)
    src = LoopTokenSource(wl.pages)
    rng = np.random.default_rng(9)
    cand = np.array([int(src.base[p]) + j for p, pg in enumerate(wl.pages) for j in range(pg.prefix_len, pg.packed_len)])
    keep = np.sort(rng.choice(cand, 400, replace=False))
    rows, o, lse, q, k, v, loop = run_loop(wl, 3, keep_rows=keep)
    assert sorted(rows.tolist()) == keep.tolist()
    # oracle decode of each kept token over its own logical rows
    sp, sh, pl, page_off, priv_off, sk, sv, pk, pv, qq = [], [], [], [], [], [], [], [], [], []
    srow = prow = 0
    for i, r in enumerate(rows):
        p = int(np.searchsorted(src.base, r, side="right") - 1)
        pg, base = wl.pages[p], int(src.base[p])
        loc = int(r) - base
        M = pg.prefix_len + pg.layout_len
        if loc < M:
            shared, priv = loc + 1, []
        else:
            kb = max(kk for kk in range(pg.num_branches) if src.ybase[p][kk] <= loc)
            shared, priv = pg.prefix_len + pg.fork_offset[kb], list(range(base + src.ybase[p][kb], int(r) + 1))
        sp.append(i); sh.append(shared); pl.append(len(priv))
        page_off.append(srow); priv_off.append(prow)
        sk.append(k[base:base + shared]); sv.append(v[base:base + shared])
        pk.append(k[priv]); pv.append(v[priv])
        srow += shared; prow += len(priv)
        qq.append(q[int(r)])
    ref_o, ref_lse = oracle.decode(np.array(sp), np.array(sh), np.array(pl), np.array(page_off), np.array(priv_off),
                                   torch.cat(sk), torch.cat(sv), torch.cat(pk), torch.cat(pv), torch.stack(qq),
                                   1.0 / math.sqrt(wl.head_dim))
    assert_close(o, lse, ref_o, ref_lse, wl.dtype)


def test_append_inputs_bit_exact():
    """The append kernel writes each K/V row to its slot and gathers the queries in order, byte for byte."""
    g = torch.Generator().manual_seed(4)
    nb, Hkv, Hq, d = 40, 2, 16, 128
    k_pool = torch.zeros((nb, Hkv, 16, d), dtype=torch.bfloat16, device=DEV)
    v_pool = torch.zeros_like(k_pool)
    rows_n = 300
    ks = torch.randn((rows_n, Hkv, d), generator=g).to(torch.bfloat16)
    vs = torch.randn((rows_n, Hkv, d), generator=g).to(torch.bfloat16)
    qs = torch.randn((rows_n, Hq, d), generator=g).to(torch.bfloat16)
    slots = np.random.default_rng(1).permutation(nb * 16)[:123].astype(np.int32)
    src = np.random.default_rng(2).integers(0, rows_n, 123).astype(np.int32)
    q_dst = torch.zeros((123, Hq, d), dtype=torch.bfloat16, device=DEV)
    pa.padoc_append_inputs(k_pool, v_pool, ks.to(DEV), vs.to(DEV), torch.from_numpy(slots).to(DEV), q_src=qs.to(DEV),
                           q_dst=q_dst, src_rows=torch.from_numpy(src).to(DEV))
    pa.padoc_check_device_errors()
    kp, vp = k_pool.cpu(), v_pool.cpu()
    for i in range(123):
        b, o = divmod(int(slots[i]), 16)
        assert torch.equal(kp[b, :, o], ks[src[i]]) and torch.equal(vp[b, :, o], vs[src[i]])
    assert torch.equal(q_dst.cpu(), qs[torch.from_numpy(src).long()])


def test_current_stream_handle():
    """The binding's default stream is torch's current stream, also inside a stream context."""
    assert pa._stream_ptr(None) == torch.cuda.current_stream().cuda_stream
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        assert pa._stream_ptr(None) == s.cuda_stream
    assert pa._stream_ptr(None) == torch.cuda.current_stream().cuda_stream
