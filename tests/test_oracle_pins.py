"""Pins of the fp64 oracle to things other than itself (CPU only).

Each test ties one oracle function to something the paper or the mathematics fixes:
  * a hand-derived visibility fixture (tests/golden/visibility_tiny.txt, Sec. 3.2 / App. C.1);
  * a simulator of Algorithm 1's mask recurrence (App. E.1), which never evaluates the ancestor
    rule itself;
  * torch's scaled_dot_product_attention and logsumexp in fp64 (library routines) over that mask;
  * the reduction to plain causal attention when N = 1 and f_1 = L (App. C.1);
  * closed forms (K = 0 gives lse = ln #visible and O = mean of visible V; one-hot V exposes the
    attention distribution; constant V is reproduced);
  * invariance under permutation of the branches;
  * the merge of partial softmax results over a partition of the keys (softmax over a union of
    disjoint key sets);
  * decode of a branch's newest token equals the matching prefill row (Algorithm 1 appends before
    it decodes).
"""
import math
import os

import numpy as np
import pytest
import torch

import oracle
from tests.alg1_sim import simulate

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rand_page(rng, P_max=24, L_max=12, N_max=5, n_max=7, allow_zero_fork=True):
    P = int(rng.integers(0, P_max + 1))
    L = int(rng.integers(0, L_max + 1))
    N = int(rng.integers(0, N_max + 1))
    lo = 0 if allow_zero_fork else min(1, L)
    forks = [int(rng.integers(lo, L + 1)) for _ in range(N)]   # ties and any order are legal
    lens = [int(rng.integers(1, n_max + 1)) for _ in range(N)]
    if P + L + sum(lens) == 0:
        P = 1
    return (P, L, forks, lens)


def _read_golden_mask(path):
    meta, rows = {}, []
    for line in open(path):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        if line[0] in "PLFN":
            key, *vals = line.split()
            meta[key] = [int(v) for v in vals]
        else:
            rows.append([int(c) for c in line])
    page = (meta["P"][0], meta["L"][0], meta["F"], meta["N"])
    return page, np.asarray(rows, np.uint8)


# --------------------------------------------------------------------------------------------
# Visibility
# --------------------------------------------------------------------------------------------

def test_dense_mask_matches_hand_derived_fixture():
    page, want = _read_golden_mask(os.path.join(GOLDEN, "visibility_tiny.txt"))
    np.testing.assert_array_equal(oracle.dense_mask([page], 0), want)


def test_alg1_simulator_matches_hand_derived_fixture():
    page, want = _read_golden_mask(os.path.join(GOLDEN, "visibility_tiny.txt"))
    np.testing.assert_array_equal(simulate(*page), want)


@pytest.mark.parametrize("seed", range(40))
def test_dense_mask_matches_alg1_recurrence(seed):
    rng = np.random.default_rng(seed)
    page = _rand_page(rng)
    np.testing.assert_array_equal(oracle.dense_mask([page], 0), simulate(*page))


def test_spans_equal_dense_rows_multi_page():
    rng = np.random.default_rng(123)
    pages = [_rand_page(rng) for _ in range(6)]
    sp = oracle.spans(pages)
    T = oracle.total_tokens(pages)
    assert sp.shape == (T, 4)
    base = 0
    for p, pg in enumerate(pages):
        m = simulate(*pg)
        S = m.shape[0]
        for r in range(S):
            row = np.zeros(T, np.uint8)
            a0, a1, b0, b1 = sp[base + r]
            assert base <= a0 <= a1 <= base + S and base <= b0 <= b1 <= base + S
            row[a0:a1] = 1
            row[b0:b1] = 1
            want = np.zeros(T, np.uint8)
            want[base:base + S] = m[r]
            np.testing.assert_array_equal(row, want)
        base += S


def test_tile_kinds_match_block_sums_of_recurrence_mask():
    rng = np.random.default_rng(7)
    pages = [_rand_page(rng, P_max=40, L_max=20, N_max=6, n_max=15) for _ in range(5)]
    T = oracle.total_tokens(pages)
    full = np.zeros((T, T), np.int64)
    base = 0
    for pg in pages:
        m = simulate(*pg)
        S = m.shape[0]
        full[base:base + S, base:base + S] = m
        base += S
    for qb, kb in [(16, 16), (8, 32), (32, 8)]:
        kinds = oracle.tile_kinds(pages, qb, kb)
        nq, nk = -(-T // qb), -(-T // kb)
        pad = np.zeros((nq * qb, nk * kb), np.int64)
        pad[:T, :T] = full
        sums = pad.reshape(nq, qb, nk, kb).sum(axis=(1, 3))
        rows = np.minimum(qb, T - np.arange(nq) * qb)[:, None]
        want = np.where(sums == 0, 0, np.where(sums == rows * kb, 2, 1))
        np.testing.assert_array_equal(kinds, want)


# --------------------------------------------------------------------------------------------
# Attention values
# --------------------------------------------------------------------------------------------

def _qkv(T, Hq, Hkv, d, seed):
    g = torch.Generator().manual_seed(seed)
    mk = lambda *s: torch.randn(*s, generator=g, dtype=torch.float32)
    return mk(T, Hq, d), mk(T, Hkv, d), mk(T, Hkv, d)


def _sdpa_reference(pages, q, k, v, scale):
    """torch SDPA (fp64) per page with the Algorithm-1 simulator's mask; GQA by consecutive groups."""
    T, Hq, d = q.shape
    Hkv = k.shape[1]
    o = torch.zeros(T, Hq, d, dtype=torch.float64)
    lse = torch.zeros(T, Hq, dtype=torch.float64)
    base = 0
    for pg in pages:
        m = torch.from_numpy(simulate(*pg).astype(bool))
        S = m.shape[0]
        qq = q[base:base + S].double().transpose(0, 1)                          # [Hq,S,d]
        kk = k[base:base + S].double().repeat_interleave(Hq // Hkv, dim=1).transpose(0, 1)
        vv = v[base:base + S].double().repeat_interleave(Hq // Hkv, dim=1).transpose(0, 1)
        o[base:base + S] = torch.nn.functional.scaled_dot_product_attention(
            qq, kk, vv, attn_mask=m, scale=scale).transpose(0, 1)
        s = (qq @ kk.transpose(1, 2)) * scale
        s = s.masked_fill(~m, float("-inf"))
        lse[base:base + S] = torch.logsumexp(s, dim=-1).transpose(0, 1)
        base += S
    return o.numpy(), lse.numpy()


@pytest.mark.parametrize("Hq,Hkv,d", [(4, 1, 8), (4, 2, 16), (3, 3, 5)])
def test_prefill_matches_sdpa_over_recurrence_mask(Hq, Hkv, d):
    rng = np.random.default_rng(Hq * 100 + Hkv * 10 + d)
    pages = [_rand_page(rng) for _ in range(4)]
    T = oracle.total_tokens(pages)
    q, k, v = _qkv(T, Hq, Hkv, d, seed=d)
    scale = 1.0 / math.sqrt(d)
    ref_o, ref_lse = _sdpa_reference(pages, q, k, v, scale)
    for fn in (oracle.prefill_dense, oracle.prefill_gather):
        o, lse = fn(pages, q, k, v, scale)
        np.testing.assert_allclose(o, ref_o, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, ref_lse, rtol=0, atol=1e-12)


def test_single_branch_full_fork_is_plain_causal_attention():
    # N = 1 and f_1 = L: the page is one causal sequence [X | layout | Y_1] (App. C.1).
    P, L, n = 37, 11, 19
    pages = [(P, L, [L], [n])]
    T = P + L + n
    Hq, Hkv, d = 4, 2, 16
    q, k, v = _qkv(T, Hq, Hkv, d, seed=5)
    scale = 0.3
    qq = q.double().transpose(0, 1)
    kk = k.double().repeat_interleave(2, dim=1).transpose(0, 1)
    vv = v.double().repeat_interleave(2, dim=1).transpose(0, 1)
    ref = torch.nn.functional.scaled_dot_product_attention(qq, kk, vv, is_causal=True, scale=scale)
    for fn in (oracle.prefill_dense, oracle.prefill_gather):
        o, _ = fn(pages, q, k, v, scale)
        np.testing.assert_allclose(o, ref.transpose(0, 1).numpy(), rtol=0, atol=1e-12)


def test_zero_keys_closed_form():
    # K = 0: every visible score is 0, so lse = ln(#visible) and O is the mean of the visible V.
    rng = np.random.default_rng(11)
    pages = [_rand_page(rng) for _ in range(4)]
    T = oracle.total_tokens(pages)
    q, _, v = _qkv(T, 2, 1, 6, seed=3)
    k = torch.zeros(T, 1, 6)
    o, lse = oracle.prefill_dense(pages, q, k, v, 0.7)
    base = 0
    for pg in pages:
        m = simulate(*pg)
        S = m.shape[0]
        cnt = m.sum(axis=1)
        np.testing.assert_allclose(lse[base:base + S], np.log(cnt)[:, None].repeat(2, 1), rtol=0, atol=1e-13)
        vv = v[base:base + S, 0].double().numpy()
        mean = (m.astype(np.float64) @ vv) / cnt[:, None]
        np.testing.assert_allclose(o[base:base + S, 0], mean, rtol=0, atol=1e-13)
        base += S


def test_one_hot_values_expose_attention_support():
    # V row j = e_j: O[q] is the attention distribution, its support must be the visible set.
    page = (6, 4, [2, 4, 0], [3, 1, 2])
    T = oracle.total_tokens([page])
    d = T
    q, k, _ = _qkv(T, 1, 1, d, seed=9)
    v = torch.eye(T).reshape(T, 1, d)
    o, _ = oracle.prefill_gather([page], q, k, v, 0.25)
    np.testing.assert_array_equal((o[:, 0] > 0).astype(np.uint8), simulate(*page))
    np.testing.assert_allclose(o[:, 0].sum(axis=1), 1.0, rtol=0, atol=1e-14)


def test_constant_values_reproduced():
    rng = np.random.default_rng(12)
    pages = [_rand_page(rng) for _ in range(3)]
    T = oracle.total_tokens(pages)
    q, k, _ = _qkv(T, 2, 2, 4, seed=1)
    v = torch.full((T, 2, 4), 0.375)
    o, _ = oracle.prefill_dense(pages, q, k, v, 1.0)
    np.testing.assert_allclose(o, 0.375, rtol=0, atol=1e-14)


def test_branch_permutation_permutes_outputs():
    P, L = 9, 7
    forks, lens = [5, 0, 7, 5], [3, 2, 4, 1]
    perm = [2, 0, 3, 1]
    pa = (P, L, forks, lens)
    pb = (P, L, [forks[i] for i in perm], [lens[i] for i in perm])
    T = oracle.total_tokens([pa])
    q, k, v = _qkv(T, 2, 1, 8, seed=4)
    ybase = [P + L + sum(lens[:i]) for i in range(4)]
    order = list(range(P + L))
    for i in perm:
        order += list(range(ybase[i], ybase[i] + lens[i]))
    o_a, l_a = oracle.prefill_dense([pa], q, k, v, 0.5)
    o_b, l_b = oracle.prefill_dense([pb], q[order], k[order], v[order], 0.5)
    np.testing.assert_array_equal(o_b, o_a[order])      # bit-identical: same per-query key order
    np.testing.assert_array_equal(l_b, l_a[order])


def _decode_case(seed, Hq=4, Hkv=2, d=16):
    rng = np.random.default_rng(seed)
    n_pages = 3
    page_len = rng.integers(1, 40, size=n_pages)
    streams = []
    for p in range(n_pages):
        for _ in range(int(rng.integers(1, 4))):
            streams.append((p, int(rng.integers(0, page_len[p] + 1)), int(rng.integers(1, 20))))
    streams.append((0, int(page_len[0]), 0))    # a layout stream: shared only, no private rows
    sp = np.array([s[0] for s in streams]); sh = np.array([s[1] for s in streams]); pl = np.array([s[2] for s in streams])
    page_off = np.concatenate([[0], np.cumsum(page_len)[:-1]])
    priv_off = np.concatenate([[0], np.cumsum(pl)[:-1]])
    g = torch.Generator().manual_seed(seed)
    sk = torch.randn(int(page_len.sum()), Hkv, d, generator=g)
    sv = torch.randn(int(page_len.sum()), Hkv, d, generator=g)
    pk = torch.randn(int(pl.sum()), Hkv, d, generator=g)
    pv = torch.randn(int(pl.sum()), Hkv, d, generator=g)
    q = torch.randn(len(streams), Hq, d, generator=g)
    return sp, sh, pl, page_off, priv_off, sk, sv, pk, pv, q


def test_decode_matches_sdpa_over_gathered_rows():
    sp, sh, pl, po, vo, sk, sv, pk, pv, q = _decode_case(21)
    o, lse = oracle.decode(sp, sh, pl, po, vo, sk, sv, pk, pv, q, 0.4)
    for s in range(len(sp)):
        kk = torch.cat([sk[po[sp[s]]:po[sp[s]] + sh[s]], pk[vo[s]:vo[s] + pl[s]]]).double()
        vv = torch.cat([sv[po[sp[s]]:po[sp[s]] + sh[s]], pv[vo[s]:vo[s] + pl[s]]]).double()
        kk = kk.repeat_interleave(2, dim=1).transpose(0, 1)      # [Hq, n, d]
        vv = vv.repeat_interleave(2, dim=1).transpose(0, 1)
        qq = q[s].double()[:, None, :]                              # [Hq, 1, d]
        ref = torch.nn.functional.scaled_dot_product_attention(qq, kk, vv, scale=0.4)[:, 0]
        np.testing.assert_allclose(o[s], ref.numpy(), rtol=0, atol=1e-12)
        ref_lse = torch.logsumexp((qq @ kk.transpose(1, 2))[:, 0] * 0.4, dim=-1)
        np.testing.assert_allclose(lse[s], ref_lse.numpy(), rtol=0, atol=1e-12)


def test_merge_of_partition_equals_unsplit_softmax():
    sp, sh, pl, po, vo, sk, sv, pk, pv, q = _decode_case(33)
    o_all, lse_all = oracle.decode(sp, sh, pl, po, vo, sk, sv, pk, pv, q, 0.4)
    S = len(sp)
    rng = np.random.default_rng(5)
    parts_o, parts_l = [], []
    # split each stream's shared rows at a random cut; the private rows are the third part
    cut = np.array([int(rng.integers(0, sh[s] + 1)) for s in range(S)])
    empty_priv = np.zeros(S, np.int64)
    z = np.zeros(S, np.int64)
    # part 1: shared rows [0, cut)
    o1, l1 = oracle.decode(sp, cut, z, po, vo, sk, sv, pk, pv, q, 0.4)
    # part 2: shared rows [cut, sh): a page offset shifted by cut, one "page" per stream
    po2 = np.array([po[sp[s]] + cut[s] for s in range(S)])
    o2, l2 = oracle.decode(np.arange(S), sh - cut, z, po2, vo, sk, sv, pk, pv, q, 0.4)
    # part 3: private rows only
    o3, l3 = oracle.decode(sp, z, pl, po, vo, sk, sv, pk, pv, q, 0.4)
    # part 4: an empty part must weigh nothing
    o4, l4 = oracle.decode(sp, z, empty_priv, po, vo, sk, sv, pk, pv, q, 0.4)
    assert np.all(np.isneginf(l4))
    R = S * q.shape[1]
    d = q.shape[2]
    po_stack = np.stack([x.reshape(R, d) for x in (o1, o2, o3, o4)])
    pl_stack = np.stack([x.reshape(R) for x in (l1, l2, l3, l4)])
    mo, ml = oracle.merge(po_stack, pl_stack)
    np.testing.assert_allclose(mo, o_all.reshape(R, d), rtol=0, atol=1e-12)
    np.testing.assert_allclose(ml, lse_all.reshape(R), rtol=0, atol=1e-12)
    # all parts empty -> lse = -inf, O = 0 (no NaN)
    eo, el = oracle.merge(np.zeros((2, 3, 4)), np.full((2, 3), -np.inf))
    assert np.all(np.isneginf(el)) and np.all(eo == 0)


def test_decode_of_newest_token_equals_prefill_row():
    # Algorithm 1 appends every live stream's input before decoding it, so branch k's decode with
    # private length n_k over the packed cache is row ybase_k + n_k - 1 of the prefill; the layout
    # stream's decode is the last layout row.
    P, L = 13, 9
    forks, lens = [3, 9, 0], [4, 6, 2]
    page = (P, L, forks, lens)
    T = oracle.total_tokens([page])
    q, k, v = _qkv(T, 4, 2, 8, seed=8)
    o_pre, l_pre = oracle.prefill_gather([page], q, k, v, 0.35)
    ybase = [P + L + sum(lens[:i]) for i in range(3)]
    rows = [ybase[i] + lens[i] - 1 for i in range(3)] + [P + L - 1]
    sp = np.zeros(4, np.int32)
    sh = np.array([P + f for f in forks] + [P + L])
    pl = np.array(lens + [0])
    po = np.array([0])
    priv_rows = sum([list(range(ybase[i], ybase[i] + lens[i])) for i in range(3)], [])
    vo = np.array([0, lens[0], lens[0] + lens[1], 0])
    o, lse = oracle.decode(sp, sh, pl, po, vo, k[:P + L], v[:P + L], k[priv_rows], v[priv_rows], q[rows], 0.35)
    np.testing.assert_allclose(o, o_pre[rows], rtol=0, atol=1e-13)
    np.testing.assert_allclose(lse, l_pre[rows], rtol=0, atol=1e-13)


def test_dense_and_gather_agree_on_workload_shapes():
    # The two formulations of App. C.1 on a scaled-down packed page with the workload's structure.
    rng = np.random.default_rng(99)
    pages = [(64, 24, [8, 16, 24], [10, 5, 13]), (40, 16, [16, 8], [7, 9]), (30, 0, [0, 0], [3, 4])]
    T = oracle.total_tokens(pages)
    q, k, v = _qkv(T, 4, 2, 16, seed=int(rng.integers(1000)))
    a = oracle.prefill_dense(pages, q, k, v, 0.25)
    b = oracle.prefill_gather(pages, q, k, v, 0.25)
    np.testing.assert_allclose(a[0], b[0], rtol=0, atol=1e-12)
    np.testing.assert_allclose(a[1], b[1], rtol=0, atol=1e-12)
