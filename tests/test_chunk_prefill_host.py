"""CPU tests of the chunked branch prefill planner (padoc_build_chunk_prefill_plan): each chunk's
tokens become consecutive streams with the visibility of Sec. 3.2 (a branch token sees its page's
shared stream before its cutoff and its own private rows up to itself; a prefix or layout token the
shared rows up to itself), and the plan reads every visible row of every token exactly once per KV
head, with the chunk's private rows on the tensor cores for chunks of 8 or more tokens."""
import numpy as np
import pytest

from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import padoc_attn as pa


@pytest.fixture(scope="module", autouse=True)
def lib():
    pbuild.build()
    return pa.load_library()


def rand_chunks(rng, n_pages):
    page_len, chunks = [], []
    for p in range(n_pages):
        pl = int(rng.integers(1, 3000))
        page_len.append(pl)
        for _ in range(int(rng.integers(0, 6))):
            n = int(rng.choice([1, 3, 7, 8, 9, 16, 31, 32, 33, 64, 100, 250]))
            if rng.random() < 0.25:       # prefix or layout tokens already on the shared stream
                if n > pl:
                    continue
                chunks.append((p, int(rng.integers(0, pl - n + 1)), -1, n))
            else:
                chunks.append((p, int(rng.integers(0, pl + 1)), int(rng.choice([0, 0, 5, 16, 130])), n))
    return np.asarray(page_len, np.int32), np.asarray(chunks, np.int32).reshape(-1, 4)


def expand(chunks):
    out = []
    for c, (p, sh, ps, n) in enumerate(chunks):
        for i in range(n):
            out.append((p, sh, ps + i + 1, c) if ps >= 0 else (p, sh + i + 1, 0, c))
    return np.asarray(out, np.int64).reshape(-1, 4)


@pytest.mark.parametrize("seed", range(10))
@pytest.mark.parametrize("tc_ctas", [0, 3])
def test_chunk_plan_covers_every_visible_row_once(seed, tc_ctas):
    rng = np.random.default_rng(700 + seed)
    page_len, chunks = rand_chunks(rng, int(rng.integers(1, 5)))
    if len(chunks) == 0:
        chunks = np.array([[0, 0, 0, 1]], np.int32)
    check_chunk_plan(page_len, chunks, tc_ctas)


def check_chunk_plan(page_len, chunks, tc_ctas, warp_ctas=0):
    Hkv = 2
    cfg = pa.make_decode_config(16, Hkv, 128, tc_ctas=tc_ctas, warp_ctas=warp_ctas)
    plan, info = pa.padoc_build_chunk_prefill_plan(page_len, chunks, cfg)
    ex = expand(chunks)
    S = len(ex)
    sp, sh, pl, ch = ex[:, 0], ex[:, 1], ex[:, 2], ex[:, 3]
    assert info.num_streams == S
    np.testing.assert_array_equal(plan[info.off_stream_page:info.off_stream_page + S], sp)
    np.testing.assert_array_equal(plan[info.off_shared_len:info.off_shared_len + S], sh)
    np.testing.assert_array_equal(plan[info.off_private_len:info.off_private_len + S], pl)
    slot_ptr = plan[info.off_slot_ptr:info.off_slot_ptr + S * Hkv + 1]
    items = plan[info.off_items:info.off_items + 8 * info.num_items].reshape(-1, 8)
    ntc = info.num_tc_items
    assert np.isin(items[:ntc, 0] & 15, [2, 3]).all() and np.isin(items[ntc:, 0], [0, 1]).all()
    assert not np.any(items[:, 0] & ~(15 | 16 | 32 | 64))
    first_of = {c: int(np.nonzero(ch == c)[0][0]) for c in range(len(chunks))}
    cov_sh = {(s, g): np.zeros(sh[s], np.int32) for s in range(S) for g in range(Hkv)}
    cov_pv = {(s, g): np.zeros(pl[s], np.int32) for s in range(S) for g in range(Hkv)}
    slots = {(s, g): [] for s in range(S) for g in range(Hkv)}
    # a piece over a group's shared and then its private rows is two items, the first flagged CONT:
    # the second is the group's private item with the same head, streams and slot, in the same CTA
    cta = plan[info.off_cta_ptr:info.off_cta_ptr + info.tc_ctas + 1] if ntc else np.zeros(1, np.int32)
    cont = (items[:, 0] & 32) != 0
    assert not cont[ntc:].any() and (ntc == 0 or not cont[ntc - 1])
    for u in np.nonzero(cont)[0]:
        a, b = items[u], items[u + 1]
        assert a[0] & 15 == 2 and b[0] & 15 == 3 and (a[2], a[5], a[6], a[7]) == (b[2], b[5], b[6], b[7])
        assert b[3] == 0, "the private part of a piece starts at the chunk's first private tile"
        assert not np.isin(u + 1, cta), "both items of a piece belong to one CTA"
    for i, (kind, idx, g, tb, te, fs, ns, slot) in enumerate(items):
        reread = bool(kind & 16)
        continued = i > 0 and cont[i - 1]
        kind &= 15
        if kind == 3:   # reread exactly when the chunk has more than one group
            assert reread == (chunks[ch[fs]][3] > 32)
        if kind == 2:   # reread exactly when the page's chunk tokens form more than one group
            assert reread == (np.count_nonzero(sp == idx) > ns)
        if kind in (2, 3):
            assert 1 <= ns <= 32 and tb % 128 == 0 and te > tb
            assert len(set(ch[fs:fs + ns])) == 1, "a tensor-core group never crosses a chunk"
        for s in range(fs, fs + ns):
            if kind == 3:        # the chunk's private rows, read through its first token's table row
                assert idx == first_of[ch[s]] and chunks[ch[s]][2] >= 0 and chunks[ch[s]][3] >= 8
                hi = min(te, pl[s])
                if hi > tb:
                    cov_pv[(s, g)][tb:hi] += 1
            elif kind == 1:
                assert s == idx
                cov_pv[(s, g)][tb:te] += 1
            else:
                assert sp[s] == idx
                hi = min(te, sh[s])
                if hi > tb:
                    cov_sh[(s, g)][tb:hi] += 1
            if not continued:    # one partial per piece
                slots[(s, g)].append(slot)
    for key in cov_sh:
        s, g = key
        assert np.all(cov_sh[key] == 1), f"shared rows of token {s} head {g}"
        assert np.all(cov_pv[key] == 1), f"private rows of token {s} head {g}"
        assert sorted(slots[key]) == list(range(slot_ptr[s * Hkv + g + 1] - slot_ptr[s * Hkv + g]))
    check_sole_and_merge_keys(plan, info, items, Hkv)


def check_sole_and_merge_keys(plan, info, items, Hkv):
    # SOLE (64): a tensor-core item that writes a partial (not the first of a chain) flagged exactly
    # when each of its streams has that one partial for its KV head; the merge joins every other key
    S, ntc = info.num_streams, info.num_tc_items
    slot_ptr = plan[info.off_slot_ptr:info.off_slot_ptr + S * Hkv + 1]
    nslots = np.diff(slot_ptr)
    cont, sole = (items[:, 0] & 32) != 0, (items[:, 0] & 64) != 0
    assert not sole[ntc:].any() and not (sole & cont).any()
    direct = set()
    for i in range(ntc):
        if cont[i]:
            continue
        _, _, g, _, _, fs, ns, _ = items[i]
        keys = [s * Hkv + g for s in range(fs, fs + ns)]
        assert bool(sole[i]) == all(nslots[k] == 1 for k in keys)
        if sole[i]:
            direct.update(keys)
    mk = plan[info.off_merge_keys:info.off_merge_keys + info.num_merge_keys]
    assert mk.tolist() == sorted(set(range(S * Hkv)) - direct)


def test_chunk_plan_validation_and_table():
    cfg = pa.make_decode_config(16, 2, 128)
    pl = np.array([100, 50], np.int32)
    pa.padoc_build_chunk_prefill_plan(pl, [[0, 100, 0, 4], [1, 40, -1, 10]], cfg)
    for bad in ([[1, 10, 0, 4], [0, 10, 0, 4]],   # pages out of order
                [[0, 101, 0, 4]],                 # cutoff past the page's shared stream
                [[1, 41, -1, 10]],                # a shared chunk reaching past the page
                [[0, 10, 0, 0]],                  # no token
                [[0, 10, -2, 3]]):
        with pytest.raises(pa.PadocError) as e:
            pa.padoc_build_chunk_prefill_plan(pl, bad, cfg)
        assert e.value.status == 1
    chunks = np.array([[0, 5, 0, 2], [0, 5, -1, 1], [1, 3, 7, 3]], np.int32)
    t = pa.padoc_expand_chunk_table(chunks, np.array([[4, 5], [0, 0], [9, 8]], np.int32), 3)
    np.testing.assert_array_equal(t, [[4, 5, -1], [4, 5, -1], [0, 0, -1], [9, 8, -1], [9, 8, -1], [9, 8, -1]])


def test_chunk_plan_properties():
    """hypothesis draws pages and chunks (1 to 70 tokens, branch chunks anywhere in a branch,
    shared-stream chunks up to the page's end, cutoffs 0 and page_len) and CTA counts; every plan
    reads each token's visible rows exactly once with consistent slots."""
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")

    @st.composite
    def cases(draw):
        n_pages = draw(st.integers(1, 3))
        page_len = [draw(st.integers(0, 700)) for _ in range(n_pages)]
        chunks = []
        for p in range(n_pages):
            for _ in range(draw(st.integers(0, 4))):
                n = draw(st.integers(1, 70))
                if page_len[p] >= n and draw(st.booleans()):
                    chunks.append((p, draw(st.integers(0, page_len[p] - n)), -1, n))
                else:
                    chunks.append((p, draw(st.integers(0, page_len[p])), draw(st.integers(0, 300)), n))
        if not chunks:
            chunks = [(0, 0, 0, 1)]
        return (np.asarray(page_len, np.int32), np.asarray(chunks, np.int32).reshape(-1, 4),
                draw(st.sampled_from([0, 1, 2, 7])), draw(st.sampled_from([0, 1, 3])))

    @hyp.settings(max_examples=80, deadline=None)
    @hyp.given(cases())
    def run(case):
        check_chunk_plan(*case)

    run()
