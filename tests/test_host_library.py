"""CPU tests of the C-ABI library: it loads, exports every declared entry point, and its host-side
C1 planners (spans, tile map, decode plan) are bit-exact against the oracle and valid."""
import os
import re

import numpy as np
import pytest

import oracle
from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import inputs
from paper_2608_06146_gb300 import padoc_attn as pa
from paper_2608_06146_gb300.inputs import PageSpec

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "padoc_attn.h")


@pytest.fixture(scope="module", autouse=True)
def lib():
    pbuild.build()
    return pa.load_library()


def _rand_pages(rng, n_pages, P_max=300, L_max=64, N_max=8, n_max=90):
    pages = []
    for _ in range(n_pages):
        P = int(rng.integers(0, P_max + 1)); L = int(rng.integers(0, L_max + 1)); N = int(rng.integers(0, N_max + 1))
        forks = [int(rng.integers(0, L + 1)) for _ in range(N)]
        lens = [int(rng.integers(1, n_max + 1)) for _ in range(N)]
        if P + L + sum(lens) == 0:
            P = 1
        pages.append(PageSpec(P, L, forks, lens))
    return pages


def test_exports_every_declared_symbol(lib):
    declared = set(re.findall(r"^\w[\w\s\*]*?\b(padoc_\w+)\s*\(", open(HEADER).read(), re.M))
    assert declared, "no declarations parsed"
    for name in declared:
        assert hasattr(lib, name), f"{name} not exported"
    assert set(pa.exported_symbols()) == declared
    assert pa.padoc_version() == 6
    assert pa.padoc_status_string(0) == "ok"


@pytest.mark.parametrize("seed", range(8))
def test_spans_bit_exact_vs_oracle(seed):
    rng = np.random.default_rng(seed)
    pages = _rand_pages(rng, int(rng.integers(1, 6)))
    np.testing.assert_array_equal(pa.padoc_build_query_spans(pages), oracle.spans(pages))


@pytest.mark.parametrize("wl_name", ["tiny", "packed_prefill"])
def test_spans_bit_exact_on_workloads(wl_name):
    wl = inputs.WORKLOADS[wl_name]()
    np.testing.assert_array_equal(pa.padoc_build_query_spans(wl.pages), oracle.spans(wl.pages))
    shuffled = inputs.packed_prefill(shuffle_branches=True)
    np.testing.assert_array_equal(pa.padoc_build_query_spans(shuffled.pages), oracle.spans(shuffled.pages))


def _dense_kinds_from_map(row_ptr, kt, kind, nqt, nkt):
    out = np.zeros((nqt, nkt), np.int8)
    for r in range(nqt):
        for e in range(row_ptr[r], row_ptr[r + 1]):
            out[r, kt[e]] = kind[e]
    return out


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("qb,kb", [(128, 128), (16, 32), (64, 16)])
def test_tile_map_bit_exact_vs_oracle_brute_force(seed, qb, kb):
    rng = np.random.default_rng(100 + seed)
    pages = _rand_pages(rng, int(rng.integers(1, 5)))
    row_ptr, kt, kind = pa.padoc_build_tile_map(pages, qb, kb)
    T = oracle.total_tokens(pages)
    want = oracle.tile_kinds(pages, qb, kb)
    nqt, nkt = want.shape
    assert len(row_ptr) == nqt + 1 and row_ptr[0] == 0 and row_ptr[-1] == len(kt)
    for r in range(nqt):   # ascending k-tiles within each q-tile
        assert np.all(np.diff(kt[row_ptr[r]:row_ptr[r + 1]]) > 0)
    np.testing.assert_array_equal(_dense_kinds_from_map(row_ptr, kt, kind, nqt, nkt), want)
    assert pa.padoc_tile_map_size(pages, qb, kb) == (nqt, len(kt))
    assert T > 0


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("qb,kb", [(32, 128), (16, 32), (64, 16)])
def test_key_tile_map_is_the_transpose_with_brute_force_kinds(seed, qb, kb):
    # the key-major map of the backward's dK/dV pass: every (q-tile, k-tile) pair of the oracle's
    # brute-force classification, listed per k-tile in ascending q-tile order; the order lists every
    # k-tile once, the longest columns first
    rng = np.random.default_rng(200 + seed)
    pages = _rand_pages(rng, int(rng.integers(1, 5)))
    col_ptr, qt, kind, order = pa.padoc_build_key_tile_map(pages, qb, kb)
    want = oracle.tile_kinds(pages, qb, kb)
    nqt, nkt = want.shape
    assert len(col_ptr) == nkt + 1 and col_ptr[0] == 0 and col_ptr[-1] == len(qt)
    got = np.zeros((nqt, nkt), np.int8)
    for c in range(nkt):
        assert np.all(np.diff(qt[col_ptr[c]:col_ptr[c + 1]]) > 0)
        got[qt[col_ptr[c]:col_ptr[c + 1]], c] = kind[col_ptr[c]:col_ptr[c + 1]]
    np.testing.assert_array_equal(got, want)
    assert sorted(order.tolist()) == list(range(nkt))
    counts = np.diff(col_ptr)[order]
    assert np.all(np.diff(counts) <= 0)
    for a, b in zip(order[:-1], order[1:]):   # ties keep ascending k-tile order
        if counts[list(order).index(a)] == counts[list(order).index(b)]:
            assert a < b
    assert pa.padoc_tile_map_size(pages, qb, kb)[1] == len(qt)


def test_prefill_bwd_tile_shapes_and_workspace():
    assert pa.padoc_prefill_bwd_tile_shapes(pa.PADOC_DTYPE_BF16, 128) == ((128, 64), (64, 128))
    assert pa.padoc_prefill_bwd_tile_shapes(pa.PADOC_DTYPE_F32, 64) == ((128, 64), (64, 128))
    with pytest.raises(pa.PadocError):
        pa.padoc_prefill_bwd_tile_shapes(pa.PADOC_DTYPE_BF16, 64)
    # lse2 and D per head, rows padded to 128
    # -lse2 and D per head and padded row, then 2 KB per padded row for the split dK/dV partials
    assert pa.padoc_prefill_bwd_workspace_size(1, 16) == 2 * 16 * 128 * 4 + 128 * 2048
    assert pa.padoc_prefill_bwd_workspace_size(32768, 16) == 2 * 16 * 32768 * 4 + 32768 * 2048
    assert pa.padoc_prefill_bwd_workspace_size(0, 4) == 0


def test_tile_map_full_size_packed_prefill_matches_interval_count():
    # 32768 tokens is too large for the quadratic brute force; count visible pairs per tile from the
    # oracle's spans with interval arithmetic instead.
    wl = inputs.packed_prefill()
    sp = oracle.spans(wl.pages)
    T = sp.shape[0]
    row_ptr, kt, kind = pa.padoc_build_tile_map(wl.pages, 128, 128)
    nqt, nkt = -(-T // 128), -(-T // 128)
    cnt = np.zeros((nqt, nkt), np.int64)
    cols = np.arange(nkt) * 128
    for s in (0, 2):
        a = sp[:, s][:, None]; b = sp[:, s + 1][:, None]
        ov = np.clip(np.minimum(b, cols + 128) - np.maximum(a, cols), 0, None)   # [T][nkt]
        np.add.at(cnt, np.arange(T) // 128, ov)
    rows = np.minimum(128, T - np.arange(nqt) * 128)[:, None]
    want = np.where(cnt == 0, 0, np.where(cnt == rows * 128, 2, 1)).astype(np.int8)
    np.testing.assert_array_equal(_dense_kinds_from_map(row_ptr, kt, kind, nqt, nkt), want)


@pytest.mark.parametrize("bad", [
    [PageSpec(10, 4, [5], [3])],          # fork offset beyond the layout stream
    [PageSpec(10, 4, [-1], [3])],         # negative fork offset
    [PageSpec(10, 4, [2], [0])],          # a branch without its branch-start token
    [PageSpec(0, 0, [], [])],             # an empty page
    [PageSpec(-1, 4, [], [])],
])
def test_malformed_pages_rejected(bad):
    with pytest.raises(pa.PadocError) as e:
        pa.padoc_build_query_spans(bad)
    assert e.value.status == 1
    with pytest.raises(pa.PadocError):
        pa.padoc_build_tile_map(bad, 128, 128)


def _plan_items(plan, info):
    items = plan[info.off_items: info.off_items + 8 * info.num_items].reshape(-1, 8)
    return items


@pytest.mark.parametrize("tc_ctas,warp_ctas", [(0, 0), (1, 1), (7, 3), (5000, 5000)])
@pytest.mark.parametrize("wl_name,layout", [("decode_page", False), ("dense_page", False), ("serving_batch", True),
                                            ("serving_batch", False), ("tiny", False)])
def test_decode_plan_covers_every_visible_token_once(wl_name, layout, tc_ctas, warp_ctas):
    check_decode_plan(inputs.WORKLOADS[wl_name](), layout, tc_ctas, warp_ctas)


def check_decode_plan(wl, layout, tc_ctas, warp_ctas):
    Hkv = wl.num_kv_heads
    cfg = pa.make_decode_config(wl.num_q_heads, Hkv, wl.head_dim, 16, layout, 0, tc_ctas, warp_ctas)
    plan, info = pa.padoc_build_decode_plan(wl.pages, cfg)
    sp, sh, pl = oracle.decode_streams(wl.pages, layout)
    S = len(sp)
    assert info.num_streams == S
    np.testing.assert_array_equal(plan[info.off_stream_page: info.off_stream_page + S], sp)
    np.testing.assert_array_equal(plan[info.off_shared_len: info.off_shared_len + S], sh)
    np.testing.assert_array_equal(plan[info.off_private_len: info.off_private_len + S], pl)
    slot_ptr = plan[info.off_slot_ptr: info.off_slot_ptr + S * Hkv + 1]
    assert slot_ptr[0] == 0 and slot_ptr[-1] == info.num_slots and np.all(np.diff(slot_ptr) >= 1)
    assert info.max_stream_slots == np.diff(slot_ptr).max()
    items = _plan_items(plan, info)
    # coverage[(stream, kv_head)] counts how often each visible token is read
    cov_sh = {(s, g): np.zeros(sh[s], np.int32) for s in range(S) for g in range(Hkv)}
    cov_pv = {(s, g): np.zeros(pl[s], np.int32) for s in range(S) for g in range(Hkv)}
    slots_used = {(s, g): [] for s in range(S) for g in range(Hkv)}
    ntc = info.num_tc_items
    kinds = items[:, 0] & 15
    assert all(kinds[:ntc] == 2) and not any(kinds[ntc:] == 2)
    assert not np.any(items[:, 0] & 16), "decode plans load every tile evict-first"
    page_streams = np.bincount(sp, minlength=len(wl.pages))
    # a page's shared stream goes to the tensor cores from 64 rows (streams x 8 query heads), or
    # from 16 in a plan with much warp work: one threshold for every page of the plan
    tc_pages = set(int(i) for i in items[:ntc, 1])
    min_rows = 16 if any(page_streams[p] * 8 < 64 for p in tc_pages) else 64
    for p in range(len(wl.pages)):
        if page_streams[p] and any(sh[s] > 0 for s in np.nonzero(sp == p)[0]):
            assert (p in tc_pages) == (page_streams[p] * 8 >= min_rows), f"page {p}"
    for kind, idx, g, tb, te, fs, ns, slot in items:
        kind &= 15
        assert tb % 16 == 0
        if kind == 2:      # tensor-core piece: whole 128-token tiles of up to 32 streams of a page
            assert 1 <= ns <= 32 and te > tb and page_streams[idx] * 8 >= min_rows and tb % 128 == 0
        elif kind == 0:    # warp item over one stream's view of the shared stream
            assert ns == 1 and te >= tb and page_streams[idx] * 8 < min_rows
        else:
            assert kind == 1 and ns == 1 and te > tb
        for s in range(fs, fs + ns):
            if kind in (0, 2):
                assert sp[s] == idx
                hi = min(te, sh[s])
                if hi > tb:
                    cov_sh[(s, g)][tb:hi] += 1
            else:
                assert s == idx
                cov_pv[(s, g)][tb:te] += 1
            slots_used[(s, g)].append(slot)
    for key in cov_sh:
        assert np.all(cov_sh[key] == 1) and np.all(cov_pv[key] == 1)
        s, g = key
        assert sorted(slots_used[key]) == list(range(slot_ptr[s * Hkv + g + 1] - slot_ptr[s * Hkv + g]))
    # the tensor-core CTAs own consecutive item ranges covering every tensor-core item once
    if ntc:
        cta = plan[info.off_cta_ptr: info.off_cta_ptr + info.tc_ctas + 1]
        assert cta[0] == 0 and cta[-1] == ntc and np.all(np.diff(cta) >= 0)
        want = tc_ctas or 152
        assert 1 <= info.tc_ctas <= want and np.all(np.diff(cta) >= 1)
        # balance: CTA loads (tiles by weight plus a fixed cost per piece) stay within one tile and
        # one piece of the average over the CTAs asked for, and none is empty
        wts = [8 if ns > 16 else 7 for *_, ns, _ in items[:ntc]]
        work = [sum(-(-(items[u, 4] - items[u, 3]) // 128) * wts[u] + (11 if wts[u] == 8 else 7)
                    for u in range(cta[c], cta[c + 1])) for c in range(info.tc_ctas)]
        if info.tc_ctas == want:
            assert max(work) <= sum(work) / want + 2 * (8 + 11)
        # lightest first: the CTAs are predicted to end in index order, which the warp planning and
        # the decode grid's pairing of warp CTAs with tensor-core CTAs rely on
        assert all(a <= b for a, b in zip(work, work[1:]))
    else:
        assert info.tc_ctas == 0
    # the warp grid: warp lists cover the warp items in order, one wave, balanced by cost
    nw_items = info.num_items - ntc
    wp = plan[info.off_warp_ptr: info.off_warp_ptr + info.num_warps + 1]
    W = 8   # warps per CTA of the warp kernel
    wctas = min(warp_ctas or 152, -(-nw_items // W))
    assert info.num_warps == min(wctas * W, nw_items)
    assert wp[0] == 0 and wp[-1] == nw_items and np.all(np.diff(wp) >= 0)
    cost = [-(-(te - tb) // 16) + 2 for _, _, _, tb, te, *_ in items[ntc:]]
    loads = np.array([sum(cost[wp[w]:wp[w + 1]]) for w in range(info.num_warps)])
    # Each warp's share follows the time it has (LPT over warps by capacity left). Without
    # tensor-core work every warp starts at once, so the shares are equal up to one item; with it,
    # the warps of one CTA start together, so their shares are equal up to one item, and the
    # longest items go to the warps that start first.
    if ntc == 0:
        assert loads.max() - loads.min() <= max(cost)
    else:
        for c in range(-(-info.num_warps // W)):
            wl_ = loads[c * W:(c + 1) * W]
            assert wl_.max() - wl_.min() <= max(cost)
        first = np.array([cost[wp[w]] if wp[w + 1] > wp[w] else 0 for w in range(info.num_warps)])
        nfree = max(0, 152 - info.tc_ctas)   # the planner's SM count on a host without a GPU
        if 0 < nfree * W < info.num_warps:
            assert first[:nfree * W].min() >= first[nfree * W:].max() - 2
    assert loads.sum() == sum(cost)
    # a warp item never reaches past its stream's cutoff (the warp kernel reads none)
    for kind, idx, g, tb, te, fs, ns, slot in items[ntc:]:
        assert te <= (sh[fs] if kind == 0 else pl[fs])
    need = pa.padoc_decode_workspace_size(info)
    # bf16 partial O and fp32 LSE per slot and query head of the group
    assert need >= info.num_slots * (wl.num_q_heads // Hkv) * (wl.head_dim * 2 + 4)
    # the merge joins every (stream, KV head) key but those a sole tensor-core item writes itself
    from tests.test_chunk_prefill_host import check_sole_and_merge_keys
    check_sole_and_merge_keys(plan, info, items, Hkv)


def test_decode_plan_properties():
    """hypothesis draws the pages (prefixes 0-3000, 0-40 branches with any fork offsets and private
    lengths 1-900, layout streams or not) and the CTA counts; every plan passes the coverage,
    slot, balance and cutoff checks above."""
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")

    @st.composite
    def cases(draw):
        pages = []
        for _ in range(draw(st.integers(1, 8))):
            P, L, N = draw(st.integers(0, 3000)), draw(st.integers(0, 300)), draw(st.integers(0, 40))
            if P + L == 0:
                P = 1
            forks = draw(st.lists(st.integers(0, L), min_size=N, max_size=N))
            lens = draw(st.lists(st.integers(1, 900), min_size=N, max_size=N))
            pages.append(PageSpec(P, L, forks, lens))
        wl = inputs.Workload("drawn", pages, 16, 2, 128, None, "decode")
        return wl, draw(st.booleans()), draw(st.sampled_from([0, 1, 5, 96])), draw(st.sampled_from([0, 1, 4, 152]))

    @hyp.settings(max_examples=60, deadline=None)
    @hyp.given(cases())
    def run(case):
        wl, layout, tc, wc = case
        if not layout and all(pg.num_branches == 0 for pg in wl.pages):
            return   # no stream at all
        check_decode_plan(wl, layout, tc, wc)

    run()


def test_decode_plan_rejects_bad_config():
    wl = inputs.decode_page()
    for cfg in [pa.make_decode_config(16, 3, 128), pa.make_decode_config(16, 2, 128, split_tokens=100),
                pa.make_decode_config(16, 2, 128, tc_ctas=-1), pa.make_decode_config(16, 2, 128, warp_ctas=-1)]:
        with pytest.raises(pa.PadocError):
            pa.padoc_build_decode_plan(wl.pages, cfg)
    with pytest.raises(pa.PadocError) as e:
        pa.padoc_build_decode_plan(wl.pages, pa.make_decode_config(16, 2, 128, block_size=32))
    assert e.value.status == 2


def test_page_array_plans_like_page_objects():
    """A persistent PageArray, updated in place between steps (every branch one token longer), plans
    exactly like page objects marshalled afresh."""
    wl = inputs.serving_batch(seed=3)
    cfg = pa.make_decode_config(16, 2, 128, tc_ctas=96, warp_ctas=152)
    arr = pa.PageArray(wl.pages)
    a, ia = pa.padoc_build_decode_plan(arr, cfg)
    b, ib = pa.padoc_build_decode_plan(wl.pages, cfg)
    np.testing.assert_array_equal(a, b)
    arr.lens += 1
    grown = [PageSpec(pg.prefix_len, pg.layout_len, list(pg.fork_offset), [n + 1 for n in pg.branch_len])
             for pg in wl.pages]
    a, _ = pa.padoc_build_decode_plan(arr, cfg)
    b, _ = pa.padoc_build_decode_plan(grown, cfg)
    np.testing.assert_array_equal(a, b)


C_PROGRAM = r"""
#include <stdio.h>
#include "padoc_attn.h"
int main(void) {
    int32_t forks[2] = {3, 8}, lens[2] = {5, 20};
    padoc_page pg = {40, 8, 2, forks, lens};
    int64_t T = 0;
    padoc_status st = padoc_packed_size(&pg, 1, &T);
    padoc_mpd *m = NULL;
    st |= padoc_mpd_create(64, 16, NULL, &m);
    int32_t pid, slots[40], news[3], lp, ls, fb;
    st |= padoc_mpd_add_page(m, 40, 2, 0, &pid, slots, news);
    st |= padoc_mpd_status(m, &lp, &ls, &fb);
    padoc_mpd_destroy(m);
    printf("%d %lld %d %d %d %s\n", (int)st, (long long)T, lp, ls, fb, padoc_status_string(PADOC_OK));
    return st != PADOC_OK;
}
"""


def test_header_is_plain_c_and_links_from_c(tmp_path):
    """The C ABI is C: the header compiles as strict C11 without CUDA's headers, and a C program
    links against the library and runs its host calls."""
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        pytest.skip("no C compiler")
    src = tmp_path / "t.c"
    src.write_text(C_PROGRAM)
    inc = os.path.dirname(HEADER)
    libdir = os.path.dirname(pbuild.LIB)
    exe = tmp_path / "t"
    subprocess.check_call(["gcc", "-std=c11", "-Wall", "-Wextra", "-Werror", "-pedantic", "-I", inc, str(src), "-L", libdir,
                           "-lpadoc_attn", f"-Wl,-rpath,{libdir}", "-o", str(exe)])
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()
    assert out == ["0", "73", "1", "3", "61", "ok"]   # 40 + 8 + 5 + 20 tokens; one page, 3 streams; 3 prefix blocks taken


def _coverage(plan, info, sp, sh, pl, Hkv):
    """every visible (stream, KV head) row read exactly once; slots 0..n-1 of each key used once"""
    S = len(sp)
    items = _plan_items(plan, info)
    slot_ptr = plan[info.off_slot_ptr: info.off_slot_ptr + S * Hkv + 1]
    cov_sh = {(s, g): np.zeros(sh[s], np.int32) for s in range(S) for g in range(Hkv)}
    cov_pv = {(s, g): np.zeros(pl[s], np.int32) for s in range(S) for g in range(Hkv)}
    used = {(s, g): [] for s in range(S) for g in range(Hkv)}
    for kind, idx, g, tb, te, fs, ns, slot in items:
        for s in range(fs, fs + ns):
            if (kind & 15) in (0, 2):
                hi = min(te, sh[s])
                if hi > tb:
                    cov_sh[(s, g)][tb:hi] += 1
            else:
                assert te <= pl[s] and te - tb <= 512
                cov_pv[(s, g)][tb:te] += 1
            used[(s, g)].append(slot)
    for (s, g) in cov_sh:
        assert np.all(cov_sh[(s, g)] == 1) and np.all(cov_pv[(s, g)] == 1)
        assert sorted(used[(s, g)]) == list(range(slot_ptr[s * Hkv + g + 1] - slot_ptr[s * Hkv + g]))


def test_advance_decode_plan_patches_lengths_and_keeps_the_work_in_place():
    wl = inputs.serving_batch(num_pages=8)
    cfg = pa.make_decode_config(16, 2, 128, 16, True, 0, 40, 40)
    plan, info = pa.padoc_build_decode_plan(wl.pages, cfg)
    plan = plan.copy()
    sp, sh, pl = oracle.decode_streams(wl.pages, True)
    before, info0 = plan.copy(), pa.padoc_decode_plan.from_buffer_copy(info)
    # nothing changed: the plan is the planner's, bit for bit
    assert pa.padoc_advance_decode_plan(plan, info, pl)
    np.testing.assert_array_equal(plan, before)
    assert bytes(info) == bytes(info0)
    # every branch grows by 1 .. 200 tokens over several steps; the layout streams keep no private rows
    rng = np.random.default_rng(3)
    cur = pl.copy()
    for step in range(6):
        grow = np.where(cur > 0, rng.integers(1, 40, size=len(cur)), 0).astype(np.int32)
        new = cur + grow
        assert pa.padoc_advance_decode_plan(plan, info, new)
        cur = new
        np.testing.assert_array_equal(plan[info.off_private_len: info.off_private_len + len(sp)], cur)
        _coverage(plan, info, sp, sh, cur, 2)
        assert info.max_stream_blocks == max(-(-int(x) // 16) for x in cur)
        assert info.kv_tokens == info0.kv_tokens + int((cur - pl).sum())
    # only the private items' ends and the private lengths moved
    items0, items1 = _plan_items(before, info0), _plan_items(plan, info)
    assert np.array_equal(items0[:, [0, 1, 2, 3, 5, 6, 7]], items1[:, [0, 1, 2, 3, 5, 6, 7]])
    moved = items0[:, 4] != items1[:, 4]
    assert np.all(items0[moved, 0] == 1)
    # the same lengths again after a full build of the grown batch: coverage holds for both
    grown = [inputs.PageSpec(pg.prefix_len, pg.layout_len, pg.fork_offset, []) for pg in wl.pages]
    s = 0
    for g, pg in zip(grown, wl.pages):
        g.branch_len = [int(x) for x in cur[s:s + pg.num_branches]]
        s += pg.num_branches + 1
    fresh, finfo = pa.padoc_build_decode_plan(grown, cfg)
    _coverage(fresh, finfo, sp, sh, cur, 2)


def test_advance_decode_plan_refuses_and_changes_nothing():
    wl = inputs.serving_batch(num_pages=4)
    cfg = pa.make_decode_config(16, 2, 128, 16, True, 0, 16, 16)
    plan, info = pa.padoc_build_decode_plan(wl.pages, cfg)
    plan = plan.copy()
    sp, sh, pl = oracle.decode_streams(wl.pages, True)
    before, info0 = plan.copy(), bytes(info)
    shorter = pl.copy(); shorter[0] -= 1
    lay = pl.copy(); lay[np.nonzero(pl == 0)[0][0]] = 1            # a layout stream has no private item
    long_ = pl.copy(); long_[0] = pl[0] + 600                        # past the warp kernel's item length
    for bad in (shorter, lay, long_):
        assert not pa.padoc_advance_decode_plan(plan, info, bad)
        np.testing.assert_array_equal(plan, before)
        assert bytes(info) == info0
    with pytest.raises(pa.PadocError):
        pa.padoc_advance_decode_plan(plan, info, pl[:-1])           # a wrong stream count


def _warp_item_cuts(plan, info):
    items = _plan_items(plan, info)[info.num_tc_items:]
    sh = {(k & 15, tb, te) for k, _, _, tb, te, *_ in items}
    return items, sh


@pytest.mark.parametrize("warp_ctas", [0, 2])
def test_planner_split_follows_warp_work(warp_ctas):
    """split_tokens 0: the warp items (shared and private) are cut every 64 tokens when the warp work
    is under 3 16-token blocks per warp of the grid, every 128 under 8, else every 256; an explicit
    split_tokens cuts the shared rows at it and private rows at 256."""
    def cuts(pages, split):
        wl = inputs.Workload("split", pages, 16, 2, 128, None, "decode")
        cfg = pa.make_decode_config(16, 2, 128, 16, False, split, 0, warp_ctas)
        plan, info = pa.padoc_build_decode_plan(wl.pages, cfg)
        items = _plan_items(plan, info)[info.num_tc_items:]
        sp, sh, pl = oracle.decode_streams(wl.pages, False)
        blocks = 2 * sum(-(-int(sh[s]) // 16) + -(-int(pl[s]) // 16) for s in range(len(sp)))   # no tensor-core page
        return items, blocks
    warps = (warp_ctas or 152) * 8
    seen = set()
    for pages in ([PageSpec(200, 0, [0], [100])], [PageSpec(600, 0, [0], [300])],
                  [PageSpec(700, 0, [0, 0], [300, 1000])], [PageSpec(3000, 0, [0] * 5, [900] * 5)] * 3,
                  [PageSpec(3000, 0, [0] * 5, [900] * 5)] * 6, [PageSpec(4000, 0, [0] * 7, [2000] * 7)] * 40):
        items, blocks = cuts(pages, 0)
        want = 64 if blocks < 3 * warps else 128 if blocks < 8 * warps else 256
        seen.add(want)
        for kind, idx, g, tb, te, *_ in items:
            assert tb % want == 0 and te - tb <= want
        assert max(te - tb for _, _, _, tb, te, *_ in items) == want
        items, _ = cuts(pages, 512)
        for kind, idx, g, tb, te, *_ in items:
            assert (tb % 512 == 0 and te - tb <= 512) if kind == 0 else (tb % 256 == 0 and te - tb <= 256)
    assert seen == {64, 128, 256}
