"""CPU tests of Algorithm 1's loop scheduler (padoc_mpd_*) and of the stream-list decode planner.

The scheduler is checked against the independent simulator of Algorithm 1's mask recurrence
(tests/alg1_sim.py, written from App. E.1's text): at every step, the rows each decoded token can
reach through its stream's cutoff, private length and block tables are exactly the simulator's
mask row of that token, and every one of those rows holds, in a host model of the pool written
only through the slots the scheduler handed out, the packed token it should hold. That pins the
fork (copy of the pre-boundary layout row), the identity extension, retirement, block reuse and
the paged addressing (C5) without a GPU.
"""
import numpy as np
import pytest

from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import padoc_attn as pa
from paper_2608_06146_gb300.inputs import LoopTokenSource, PageSpec
from tests.alg1_sim import simulate

BS = 16


@pytest.fixture(scope="module", autouse=True)
def lib():
    pbuild.build()
    return pa.load_library()


def _rand_pages(rng, n_pages, P_max=40, L_max=12, N_max=5, n_max=20):
    pages = []
    for _ in range(n_pages):
        P = int(rng.integers(0, P_max + 1)); L = int(rng.integers(0, L_max + 1)); N = int(rng.integers(0, N_max + 1))
        forks = [int(rng.integers(0, L + 1)) for _ in range(N)]   # any order, ties, f = 0 and f = L allowed
        lens = [int(rng.integers(1, n_max + 1)) for _ in range(N)]
        pages.append(PageSpec(P, L, forks, lens))
    return pages


def _blocks_needed(pages):
    return sum(-(-(pg.prefix_len + pg.layout_len) // BS) + sum(-(-n // BS) for n in pg.branch_len) for pg in pages)


def run_loop(pages, num_blocks, block_order=None, admit_at=None, check=True):
    """Runs the loop to the end with the synthetic token source, checking every step against the
    simulator. admit_at[p] = step before which page p is admitted (default: all at step 0).
    Returns (decoded packed rows in order, steps, scheduler)."""
    src = LoopTokenSource(pages)
    mpd = pa.Mpd(num_blocks, BS, block_order)
    sims = [simulate(pg.prefix_len, pg.layout_len, pg.fork_offset, pg.branch_len) for pg in pages]
    pool = {}                      # slot -> packed row written there
    admit_at = admit_at or [0] * len(pages)
    decoded = []
    step = 0
    pending = sorted(range(len(pages)), key=lambda p: admit_at[p])
    page_of_id = {}
    while True:
        while pending and admit_at[pending[0]] <= step:
            p = pending.pop(0)
            P, nf, leos, rows = src.admission(p)
            pid, slots, new = mpd.add_page(P, nf, leos)
            page_of_id[pid] = p
            src.admitted(p, new)
            for s, r in zip(slots, rows):
                pool[int(s)] = int(r)
        lp, ls, fb = mpd.status()
        if ls == 0:
            if not pending:
                break
            step += 1
            continue
        ids, slots = mpd.begin_step()
        rows = src.rows(ids)
        for s, r in zip(slots, rows):
            pool[int(s)] = int(r)
        page_len, streams, pt, st = mpd.step_tables()
        assert len(streams) == len(ids)
        for i, sid in enumerate(ids):
            q = src.token_row(int(sid))
            decoded.append(q)
            if not check:
                continue
            p, k = src.stream_of(int(sid))
            pg, base = pages[p], int(src.base[p])
            sh, pr = int(streams[i]["shared_len"]), int(streams[i]["private_len"])
            pi = int(streams[i]["page"])
            assert sh <= page_len[pi]
            vis = set()
            for j in range(sh):   # shared stream rows through the page table
                slot = int(pt[pi, j // BS]) * BS + j % BS
                assert pool[slot] == base + j, "shared row holds the wrong token"
                vis.add(j)
            for j in range(pr):   # private rows through the stream table
                slot = int(st[i, j // BS]) * BS + j % BS
                want = base + src.ybase[p][k] + j
                assert pool[slot] == want, "private row holds the wrong token"
                vis.add(src.ybase[p][k] + j)
            if k < 0:
                assert pr == 0
            want_vis = set(np.nonzero(sims[p][q - base])[0].tolist())
            assert vis == want_vis, f"page {p} token {q - base}: visible set differs from Algorithm 1's mask row"
        nf, eos = src.events(ids)
        new = mpd.end_step(nf, eos)
        src.forked(ids, nf, new)
        step += 1
    return decoded, step, mpd


@pytest.mark.parametrize("seed", range(12))
def test_loop_matches_alg1_recurrence(seed):
    rng = np.random.default_rng(100 + seed)
    pages = _rand_pages(rng, int(rng.integers(1, 5)))
    need = _blocks_needed(pages)
    order = rng.permutation(need + 3).astype(np.int32)
    decoded, steps, mpd = run_loop(pages, need + 3, order)
    src = LoopTokenSource(pages)
    # every layout and branch token is decoded exactly once; prefix tokens are prefilled, not decoded
    want = sorted(int(src.base[p]) + j for p, pg in enumerate(pages) for j in range(pg.prefix_len, pg.packed_len))
    assert sorted(decoded) == want
    assert mpd.status() == (0, 0, need + 3)   # every block is back in the pool


def test_loop_staggered_admission_and_block_reuse():
    """Pages admitted while others decode, in a pool just large enough for the peak: blocks of
    retired branches are handed out again and never alias a row still visible."""
    rng = np.random.default_rng(7)
    pages = _rand_pages(rng, 6, P_max=60, L_max=16, N_max=6, n_max=40)
    admit = [0, 0, 3, 9, 20, 21]
    # smallest pool that runs to the end
    lo, hi = 1, _blocks_needed(pages)
    while lo < hi:
        mid = (lo + hi) // 2
        try:
            run_loop(pages, mid, admit_at=admit, check=False)
            hi = mid
        except pa.PadocError as e:
            assert e.status == 6   # capacity
            lo = mid + 1
    assert lo < _blocks_needed(pages), "the loop should reuse retired blocks"
    run_loop(pages, lo, admit_at=admit)


def test_fork_at_prefill_and_layout_eos_at_once():
    """f = 0 branches fork from the prefill's output; L = 0 retires the layout stream at once; a page
    with neither returns its prefix blocks immediately."""
    pages = [PageSpec(5, 0, [0, 0], [3, 1]), PageSpec(17, 4, [0, 4, 4, 2], [2, 5, 1, 1]), PageSpec(0, 3, [3], [2])]
    decoded, steps, mpd = run_loop(pages, 16)
    assert steps == 4 + 5   # the layout stream's 4 tokens, then the 5 of the branch forked at its last one
    m = pa.Mpd(4)
    pid, slots, new = m.add_page(20, 0, True)
    assert new.tolist() == [-1] and m.status() == (0, 0, 4)


def test_capacity_errors_leave_state_unchanged():
    m = pa.Mpd(2, BS, np.array([1, 0], np.int32))
    with pytest.raises(pa.PadocError) as e:
        m.add_page(33)
    assert e.value.status == 6 and m.status() == (0, 0, 2)
    pid, slots, new = m.add_page(16, 1)       # one block for the prefix; the branch forks at f = 0
    assert slots.tolist() == list(range(16, 32)) and m.status() == (1, 2, 1)


def test_capacity_on_begin_step():
    m = pa.Mpd(2, BS, np.array([1, 0], np.int32))
    m.add_page(16, 1)
    before = m.status()
    with pytest.raises(pa.PadocError) as e:
        m.begin_step()
    assert e.value.status == 6 and m.status() == before
    with pytest.raises(pa.PadocError):        # no step was begun
        m.end_step(np.zeros(2, np.int32), np.zeros(2, np.uint8))


def test_event_validation():
    m = pa.Mpd(8)
    m.add_page(3, 1)
    ids, slots = m.begin_step()
    assert len(ids) == 2                       # the branch first, then the layout stream
    with pytest.raises(pa.PadocError) as e:
        m.end_step(np.array([1, 0], np.int32), np.zeros(2, np.uint8))   # a branch cannot fork
    assert e.value.status == 1
    with pytest.raises(pa.PadocError):
        m.end_step(np.zeros(3, np.int32), np.zeros(3, np.uint8))       # wrong stream count
    with pytest.raises(pa.PadocError):
        m.add_page(4)                                                   # no admission inside a step
    new = m.end_step(np.array([0, 2], np.int32), np.array([1, 1], np.uint8))   # fork two, retire both
    assert len(new) == 2 and m.status()[:2] == (1, 2)
    ids, slots = m.begin_step()
    page_len, streams, pt, st = m.step_tables()
    assert page_len.tolist() == [4] and [(int(s["shared_len"]), int(s["private_len"])) for s in streams] == [(4, 1), (4, 1)]


# ------------------------------------------------------------------------------------------------
# The stream-list planner gives the page planner's plan for the same streams
# ------------------------------------------------------------------------------------------------

def _streams_of(pages, layout):
    out, page_len = [], []
    for p, pg in enumerate(pages):
        page_len.append(pg.prefix_len + pg.layout_len)
        for f, n in zip(pg.fork_offset, pg.branch_len):
            out.append((p, pg.prefix_len + f, n))
        if layout:
            out.append((p, pg.prefix_len + pg.layout_len, 0))
    return np.asarray(page_len, np.int32), np.asarray(out, np.int32).reshape(-1, 3)


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("layout", [False, True])
def test_stream_list_plan_equals_page_plan(seed, layout):
    rng = np.random.default_rng(300 + seed)
    pages = []
    for _ in range(int(rng.integers(1, 12))):
        P = int(rng.integers(1, 3000)); N = int(rng.integers(0, 40)); L = 8 * N + int(rng.integers(0, 3))
        pages.append(PageSpec(P, L, [int(rng.integers(0, L + 1)) for _ in range(N)],
                              [int(rng.integers(1, 700)) for _ in range(N)]))
    cfg = pa.make_decode_config(16, 2, 128, layout_streams=layout, tc_ctas=96, warp_ctas=152)
    a, ia = pa.padoc_build_decode_plan(pages, cfg)
    page_len, streams = _streams_of(pages, layout)
    cfg2 = pa.make_decode_config(16, 2, 128, layout_streams=False, tc_ctas=96, warp_ctas=152)
    b, ib = pa.padoc_build_decode_plan_streams(page_len, streams, cfg2)
    np.testing.assert_array_equal(a, b)
    for f in ("num_streams", "num_items", "num_tc_items", "tc_ctas", "num_warps", "num_slots", "max_page_blocks",
              "max_stream_blocks", "kv_tokens"):
        assert getattr(ia, f) == getattr(ib, f), f


def test_stream_list_validation():
    cfg = pa.make_decode_config(16, 2, 128)
    ok = np.array([[0, 10, 1], [1, 5, 2]], np.int32)
    pa.padoc_build_decode_plan_streams(np.array([10, 5], np.int32), ok, cfg)
    for bad_pl, bad in [([10, 5], [[1, 5, 2], [0, 10, 1]]),    # pages out of order
                        ([10, 5], [[0, 11, 1]]),                # cutoff past the page's shared stream
                        ([10, 5], [[2, 1, 1]]),                 # no such page
                        ([10, 5], [[0, 0, 0]])]:                # nothing visible
        with pytest.raises(pa.PadocError) as e:
            pa.padoc_build_decode_plan_streams(np.array(bad_pl, np.int32), np.array(bad, np.int32), cfg)
        assert e.value.status == 1
    with pytest.raises(pa.PadocError):   # the list names every stream: layout_streams must be 0
        pa.padoc_build_decode_plan_streams(np.array([10, 5], np.int32), ok,
                                           pa.make_decode_config(16, 2, 128, layout_streams=True))




def check_first_blocks(stage, st, plan, info, page_len, streams, pt, stt, Hkv=2):
    """The step's first-block rows: for each warp list, the pool rows of its first item's first four
    blocks, read from that item's block-table row, -2 - row for the block holding the stream's
    newest row (the last shared row of the page for a shared item, the last private row for a
    private one), -1 past the item's end."""
    W = info.num_warps
    fb = stage[st.off_first_blocks:st.off_first_blocks + 4 * W].reshape(W, 4)
    wp = plan[info.off_warp_ptr:info.off_warp_ptr + W + 1]
    items = plan[info.off_items:info.off_items + 8 * info.num_items].reshape(-1, 8)[info.num_tc_items:]
    for w in range(W):
        want = [-1] * 4
        if wp[w] < wp[w + 1]:
            kind, idx, g, tb, te, fs, ns, slot = items[wp[w]]
            row, hot = (pt[idx], (page_len[idx] - 1) // BS) if kind == 0 else (stt[fs], (streams[fs]["private_len"] - 1) // BS)
            nb = -(-(te - tb) // BS) if te > tb else 0
            for k in range(min(4, nb)):
                r = (int(row[tb // BS + k]) * Hkv + int(g)) * BS
                want[k] = -2 - r if tb // BS + k == hot else r
        assert fb[w].tolist() == want, f"warp {w}"


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("ctas", [(96, 152), (0, 0), "alternating"])
def test_prepare_step_equals_granular_calls(seed, ctas):
    """padoc_mpd_prepare_step writes exactly what begin_step, step_tables and the stream-list planner
    give, step after step, for two schedulers driven by the same events (the scheduler keeps its
    planner's arrays and its last tensor-core bound search from step to step; each comparison plan
    is built from nothing; "alternating" changes the CTA counts asked for at every step)."""
    rng = np.random.default_rng(500 + seed)
    pages = _rand_pages(rng, int(rng.integers(2, 6)), P_max=300, L_max=40, N_max=12, n_max=70)
    nb = _blocks_needed(pages) + 5
    order = rng.permutation(nb).astype(np.int32)
    cfgs = [pa.make_decode_config(16, 2, 128, tc_ctas=t, warp_ctas=w)
            for t, w in ([(96, 152), (40, 0), (0, 0)] if ctas == "alternating" else [ctas])]
    step_no = 0
    a, b = pa.Mpd(nb, BS, order), pa.Mpd(nb, BS, order)
    src = LoopTokenSource(pages)
    for p in range(len(pages)):
        P, nf, leos, _ = src.admission(p)
        a.add_page(P, nf, leos)
        _, _, new = b.add_page(P, nf, leos)
        src.admitted(p, new)
    stage = np.zeros(16, np.int32)
    while b.status()[1] > 0:
        cfg = cfgs[step_no % len(cfgs)]
        step_no += 1
        try:
            st = a.prepare_step(cfg, stage)
        except pa.PadocError as e:
            assert e.status == 6 and e.step.total_words > stage.size
            assert a.status() == b.status(), "a too-small stage begins nothing"
            stage = np.zeros(int(e.step.total_words), np.int32)
            st = a.prepare_step(cfg, stage)
        ids, slots = b.begin_step()
        page_len, streams, pt, stt = b.step_tables()
        plan, info = pa.padoc_build_decode_plan_streams(page_len, streams, cfg)
        C = st.num_streams
        assert C == len(ids) and st.num_pages == len(page_len)
        np.testing.assert_array_equal(stage[st.off_stream_ids:st.off_stream_ids + C], ids)
        np.testing.assert_array_equal(stage[st.off_slots:st.off_slots + C], slots)
        np.testing.assert_array_equal(stage[st.off_plan:st.off_plan + st.plan.plan_ints], plan)
        np.testing.assert_array_equal(
            stage[st.off_page_table:st.off_page_table + st.num_pages * st.page_stride].reshape(-1, st.page_stride), pt)
        np.testing.assert_array_equal(
            stage[st.off_stream_table:st.off_stream_table + C * st.stream_stride].reshape(-1, st.stream_stride), stt)
        for off in (st.off_page_table, st.off_stream_table, st.off_slots, st.off_rows, st.off_first_blocks,
                    st.off_stream_ids):
            assert off % 32 == 0
        assert st.plan.num_items == info.num_items and st.plan.num_slots == info.num_slots
        check_first_blocks(stage, st, plan, info, page_len, streams, pt, stt)
        src.rows(ids)
        nf, eos = src.events(ids)
        new = b.end_step(nf, eos)
        np.testing.assert_array_equal(a.end_step(nf, eos), new)
        src.forked(ids, nf, new)
    assert a.status() == b.status() == (0, 0, nb)


def test_launch_step_validates_before_any_device_work(lib):
    """padoc_mpd_launch_step rejects a device buffer too small for the stage, not 256-byte aligned or
    null, and a null pool, before it touches the device (these checks need no GPU)."""
    import ctypes
    m = pa.Mpd(64)
    m.add_page(40, 2)
    cfg = pa.make_decode_config(16, 2, 128)
    stage = np.zeros(1 << 16, np.int32)
    st = m.prepare_step(cfg, stage)
    assert st.num_streams == 3 and st.upload_words > 0
    pool = pa.padoc_kv_pool(256, 512, 64, 16, 2, 128, pa.PADOC_DTYPE_BF16)   # never dereferenced here
    sp = stage.ctypes.data
    call = lambda stage_p, dev, cap, pool_p: lib.padoc_mpd_launch_step(
        ctypes.byref(st), stage_p, dev, cap, pool_p, 1024, 1024, 1024, 10, 1024, 0.1, 1024, 1024, 1024, 1 << 20, None)
    assert call(sp, 4096, st.upload_words - 1, ctypes.byref(pool)) == 1   # too small
    assert call(sp, 4096 + 4, st.upload_words, ctypes.byref(pool)) == 1   # not 256-byte aligned
    assert call(sp, None, st.upload_words, ctypes.byref(pool)) == 1       # no device buffer
    assert call(sp, 4096, st.upload_words, None) == 1                     # no pool
    m.end_step(np.zeros(3, np.int32), np.zeros(3, np.uint8))


def test_runner_validates_before_any_device_work(lib):
    """padoc_mpd_runner_create rejects a configuration or pool that does not fit the scheduler before
    any CUDA call; without a GPU, a valid one fails with the CUDA status, loudly; a runner step
    checks its arguments before it begins anything (these checks need no GPU)."""
    import ctypes
    m = pa.Mpd(64)
    cfg = pa.make_decode_config(16, 2, 128)
    h = ctypes.c_void_p()
    mk = lambda nb, bs, hkv, d: pa.padoc_kv_pool(256, 512, nb, bs, hkv, d, pa.PADOC_DTYPE_BF16)
    for pool in (mk(63, 16, 2, 128), mk(64, 8, 2, 128), mk(64, 16, 1, 128), mk(64, 16, 2, 64)):
        assert lib.padoc_mpd_runner_create(m._h, ctypes.byref(cfg), ctypes.byref(pool), ctypes.byref(h)) == 1
    lay = pa.make_decode_config(16, 2, 128, True)
    assert lib.padoc_mpd_runner_create(m._h, ctypes.byref(lay), ctypes.byref(mk(64, 16, 2, 128)), ctypes.byref(h)) == 1
    assert lib.padoc_mpd_runner_create(None, ctypes.byref(cfg), ctypes.byref(mk(64, 16, 2, 128)), ctypes.byref(h)) == 1
    assert lib.padoc_mpd_runner_step(None, None, None, None) == 1
    import torch
    if not torch.cuda.is_available():
        with pytest.raises(pa.PadocError) as e:
            pa.MpdRunner(m, cfg, mk(64, 16, 2, 128))
        assert e.value.status == 4
