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
  * the backward: central differences of the forward, torch autograd through the per-branch
    gather (whose backward scatter-adds onto the shared rows, App. C.1), the page sums that the
    softmax fixes (sum of dK is zero, sum of dV is the sum of dO) and the K = 0 closed form.
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
    sp, sh, pl = oracle.decode_streams([page], layout_streams=True)
    np.testing.assert_array_equal(sp, np.zeros(4, np.int32))
    po = np.array([0])
    priv_rows = sum([list(range(ybase[i], ybase[i] + lens[i])) for i in range(3)], [])
    vo = np.array([0, lens[0], lens[0] + lens[1], 0])
    o, lse = oracle.decode(sp, sh, pl, po, vo, k[:P + L], v[:P + L], k[priv_rows], v[priv_rows], q[rows], 0.35)
    np.testing.assert_allclose(o, o_pre[rows], rtol=0, atol=1e-13)
    np.testing.assert_allclose(lse, l_pre[rows], rtol=0, atol=1e-13)


@pytest.mark.parametrize("seed", range(6))
def test_decode_streams_equal_dense_mask_rows_of_newest_tokens(seed):
    # The per-stream decode plan {page, shared_len, private_len} against the dense visibility built
    # from node membership: the newest token of branch k sees exactly the first shared_len columns
    # of its page's shared stream and private_len columns of its own segment; the layout stream's
    # newest token sees the whole shared stream and nothing else.
    rng = np.random.default_rng(seed)
    pages = []
    for _ in range(3):
        P, L, n = int(rng.integers(0, 20)), int(rng.integers(0, 9)), int(rng.integers(1, 5))
        if P + L == 0:
            P = 1
        pages.append((P, L, [int(x) for x in rng.integers(0, L + 1, size=n)], [int(x) for x in rng.integers(1, 6, size=n)]))
    sp, sh, pl = oracle.decode_streams(pages, layout_streams=True)
    s = 0
    for p, (P, L, forks, lens) in enumerate(pages):
        m = oracle.dense_mask(pages, p)
        ybase = P + L
        for k, n in enumerate(lens):
            row = m[ybase + n - 1]
            assert sp[s] == p and pl[s] == n
            assert row[:P + L].sum() == sh[s] and row[:sh[s]].all()
            assert row[ybase:ybase + n].all() and row.sum() == sh[s] + n
            ybase += n
            s += 1
        row = m[P + L - 1]
        assert sp[s] == p and pl[s] == 0 and sh[s] == P + L and row.sum() == P + L
        s += 1
    assert s == len(sp)


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


# --------------------------------------------------------------------------------------------
# Backward (gradients of the packed prefill)
# --------------------------------------------------------------------------------------------

def _grid_inputs(rng, T, Hq, Hkv, d, step=2.0 ** -12):
    """Inputs on a 2^-12 grid in [-1, 1): x +- 2^-10 stays exact in fp32, so central differences
    of the fp64 forward see exactly the perturbed values."""
    f = lambda *s: (np.round(rng.uniform(-1, 1, s) / step) * step).astype(np.float32)
    return f(T, Hq, d), f(T, Hkv, d), f(T, Hkv, d), f(T, Hq, d)


def test_prefill_bwd_matches_central_differences_of_forward():
    """dQ, dK, dV are the derivatives of L = sum(dO * O) with O from the (separately pinned)
    forward: central differences with h = 2^-10 (error O(h^2) ~ 1e-6)."""
    pages = [(3, 2, [1, 2], [2, 1]), (2, 1, [0], [2])]
    rng = np.random.default_rng(7)
    T = oracle.total_tokens(pages)
    Hq, Hkv, d, scale = 4, 2, 3, 0.7
    q, k, v, g = _grid_inputs(rng, T, Hq, Hkv, d)
    dq, dk, dv = oracle.prefill_bwd(pages, q, k, v, g, scale)
    h = 2.0 ** -10

    def loss(qq, kk, vv):
        o, _ = oracle.prefill_dense(pages, qq, kk, vv, scale)
        return float((o * g.astype(np.float64)).sum())

    for name, arr, got in (("q", q, dq), ("k", k, dk), ("v", v, dv)):
        fd = np.zeros(arr.shape)
        for idx in np.ndindex(arr.shape):
            a = arr.copy(); a[idx] += np.float32(h)
            b = arr.copy(); b[idx] -= np.float32(h)
            args = {"q": (q, k, v), "k": (q, k, v), "v": (q, k, v)}[name]
            pa = [a if x is arr else x for x in args]
            pb = [b if x is arr else x for x in args]
            fd[idx] = (loss(*pa) - loss(*pb)) / (2 * h)
        np.testing.assert_allclose(got, fd, rtol=0, atol=2e-5 * max(1.0, np.abs(fd).max()), err_msg=name)


def _gather_autograd(pages, q, k, v, g, scale):
    """The paper's tree-varlen formulation in torch fp64 with autograd: the shared stream is one
    causal problem; branch k gathers [M_<P+f_k ; Y_k] with index_select and runs bottom-right
    causal attention; the gather's backward scatter-adds onto the shared rows (App. C.1). The
    masks are built here from (P, L, f, n) alone."""
    Q = torch.tensor(q, dtype=torch.float64, requires_grad=True)
    K = torch.tensor(k, dtype=torch.float64, requires_grad=True)
    V = torch.tensor(v, dtype=torch.float64, requires_grad=True)
    G = torch.tensor(g, dtype=torch.float64)
    T, Hq, d = q.shape
    rep = Hq // k.shape[1]
    out = torch.zeros(T, Hq, d, dtype=torch.float64)

    def attend(qrows, krows, n_q, n_k):
        qq = Q.index_select(0, qrows).transpose(0, 1)                           # [Hq, n_q, d]
        kk = K.index_select(0, krows).repeat_interleave(rep, 1).transpose(0, 1)  # [Hq, n_k, d]
        vv = V.index_select(0, krows).repeat_interleave(rep, 1).transpose(0, 1)
        i = torch.arange(n_q)[:, None]
        j = torch.arange(n_k)[None, :]
        allowed = j <= i + (n_k - n_q)                                           # bottom-right causal
        s = (qq @ kk.transpose(1, 2)) * scale
        s = s.masked_fill(~allowed, float("-inf"))
        return (torch.softmax(s, -1) @ vv).transpose(0, 1)

    base = 0
    for P, L, f, n in pages:
        M = P + L
        rows = []
        if M:
            idx = torch.arange(base, base + M)
            rows.append((idx, attend(idx, idx, M, M)))
        y = base + M
        for fk, nk in zip(f, n):
            qi = torch.arange(y, y + nk)
            ki = torch.cat([torch.arange(base, base + P + fk), qi])
            rows.append((qi, attend(qi, ki, nk, P + fk + nk)))
            y += nk
        for idx, o in rows:
            out = out.index_put((idx,), o)
        base = y
    (out * G).sum().backward()
    return Q.grad.numpy(), K.grad.numpy(), V.grad.numpy()


@pytest.mark.parametrize("seed", range(6))
def test_prefill_bwd_matches_torch_autograd_of_gather(seed):
    rng = np.random.default_rng(100 + seed)
    pages = [_rand_page(rng, P_max=12, L_max=8, N_max=4, n_max=5) for _ in range(3)]
    T = oracle.total_tokens(pages)
    Hq, Hkv, d = [(2, 1, 8), (4, 2, 4), (6, 3, 5)][seed % 3]
    q = rng.standard_normal((T, Hq, d)).astype(np.float32)
    k = rng.standard_normal((T, Hkv, d)).astype(np.float32)
    v = rng.standard_normal((T, Hkv, d)).astype(np.float32)
    g = rng.standard_normal((T, Hq, d)).astype(np.float32)
    scale = 1 / math.sqrt(d)
    dq, dk, dv = oracle.prefill_bwd(pages, q, k, v, g, scale)
    tq, tk, tv = _gather_autograd(pages, q, k, v, g, scale)
    for got, want in ((dq, tq), (dk, tk), (dv, tv)):
        np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-11)


def test_prefill_bwd_page_sums_and_first_token():
    """Per page and KV head: sum_j dK_j = 0 (every query's dS row sums to zero) and
    sum_j dV_j = sum of the group's dO rows (every query's P row sums to one); a page's first
    token sees only itself, so its dQ is zero."""
    rng = np.random.default_rng(5)
    pages = [(9, 6, [2, 6, 0], [4, 3, 2]), (1, 0, [], []), (5, 3, [3, 1], [1, 6])]
    T = oracle.total_tokens(pages)
    Hq, Hkv, d = 4, 2, 6
    q = rng.standard_normal((T, Hq, d)).astype(np.float32)
    k = rng.standard_normal((T, Hkv, d)).astype(np.float32)
    v = rng.standard_normal((T, Hkv, d)).astype(np.float32)
    g = rng.standard_normal((T, Hq, d)).astype(np.float32)
    dq, dk, dv = oracle.prefill_bwd(pages, q, k, v, g, 0.5)
    base = 0
    for P, L, f, n in pages:
        S = P + L + sum(n)
        sl = slice(base, base + S)
        np.testing.assert_allclose(dk[sl].sum(0), 0.0, atol=1e-12)
        want = g[sl].astype(np.float64).reshape(S, Hkv, Hq // Hkv, d).sum((0, 2))
        np.testing.assert_allclose(dv[sl].sum(0), want, rtol=1e-12, atol=1e-12)
        np.testing.assert_array_equal(dq[base], 0.0)
        base += S


def test_prefill_bwd_zero_keys_closed_form():
    """K = 0 makes every visible weight 1/n_i: dV_j = sum over queries i that see j of dO_i / n_i
    (summed over the group's heads), dQ = 0, and
    dK_j = scale * sum_i (1/n_i) (dO_i.v_j - mean over i's visible keys of dO_i.v) q_i."""
    rng = np.random.default_rng(11)
    pages = [(6, 4, [4, 1], [3, 2]), (3, 2, [2], [3])]
    T = oracle.total_tokens(pages)
    Hq, Hkv, d, scale = 2, 1, 5, 0.3
    q = rng.standard_normal((T, Hq, d)).astype(np.float32)
    k = np.zeros((T, Hkv, d), np.float32)
    v = rng.standard_normal((T, Hkv, d)).astype(np.float32)
    g = rng.standard_normal((T, Hq, d)).astype(np.float32)
    dq, dk, dv = oracle.prefill_bwd(pages, q, k, v, g, scale)
    sp = oracle.spans(pages)
    vis = np.zeros((T, T), bool)
    for t in range(T):
        vis[t, sp[t, 0]:sp[t, 1]] = True
        vis[t, sp[t, 2]:sp[t, 3]] = True
    n = vis.sum(1)
    q64, v64, g64 = (x.astype(np.float64) for x in (q, v, g))
    want_dv = np.zeros((T, Hkv, d))
    want_dk = np.zeros((T, Hkv, d))
    for i in range(T):
        for h in range(Hq):
            dp = v64[:, 0, :] @ g64[i, h]                 # dO_i . v_j for every j
            mean = dp[vis[i]].mean()
            for j in np.nonzero(vis[i])[0]:
                want_dv[j, 0] += g64[i, h] / n[i]
                want_dk[j, 0] += scale * (dp[j] - mean) / n[i] * q64[i, h]
    np.testing.assert_array_equal(dq, 0.0)
    np.testing.assert_allclose(dv, want_dv, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(dk, want_dk, rtol=1e-10, atol=1e-12)


def test_prefill_bwd_row_selection_matches_full():
    rng = np.random.default_rng(3)
    pages = [(7, 4, [1, 4], [3, 2]), (4, 2, [2, 0], [2, 2])]
    T = oracle.total_tokens(pages)
    q = rng.standard_normal((T, 2, 4)).astype(np.float32)
    k = rng.standard_normal((T, 1, 4)).astype(np.float32)
    v = rng.standard_normal((T, 1, 4)).astype(np.float32)
    g = rng.standard_normal((T, 2, 4)).astype(np.float32)
    full = oracle.prefill_bwd(pages, q, k, v, g, 0.5)
    qr, kr = [T - 1, 0, 5, 12], [3, T - 2, 0]
    part = oracle.prefill_bwd(pages, q, k, v, g, 0.5, q_rows=qr, k_rows=kr)
    np.testing.assert_array_equal(part[0], full[0][qr])
    np.testing.assert_array_equal(part[1], full[1][kr])
    np.testing.assert_array_equal(part[2], full[2][kr])


# ------------------------------------------------------------------------------------------------
# FP8 (E4M3) KV cache
# ------------------------------------------------------------------------------------------------

def test_e4m3_decode_matches_torch_on_every_code():
    """All 256 codes against torch's float8_e4m3fn (a library decoder of the same format)."""
    codes = np.arange(256, dtype=np.uint8)
    ref = torch.from_numpy(codes.copy()).view(torch.float8_e4m3fn).to(torch.float64).numpy()
    got = oracle.e4m3_decode(codes)
    assert np.array_equal(np.isnan(got), np.isnan(ref))
    ok = ~np.isnan(ref)
    np.testing.assert_array_equal(got[ok], ref[ok])
    np.testing.assert_array_equal(np.signbit(got[ok]), np.signbit(ref[ok]))
    assert np.nanmax(got) == 448.0 and got[1] == 2.0 ** -9


def test_e4m3_encode_matches_torch_rounding_in_range():
    """Nearest-even encoding against torch's conversion wherever torch's result is finite (|x| < 464):
    random values over the whole range, exact midpoints between neighbouring codes (ties), the
    subnormal range and signed zeros."""
    rng = np.random.default_rng(0)
    vals = oracle.e4m3_decode(np.arange(0, 0x7E, dtype=np.uint8))
    mids = (vals[:-1] + vals[1:]) / 2
    x = np.concatenate([rng.uniform(-463, 463, 20000), np.exp(rng.uniform(-14, 6, 20000)) * rng.choice([-1, 1], 20000),
                        mids, -mids, vals, [0.0, -0.0, 2.0 ** -10, 3 * 2.0 ** -10, 447.9, 463.9]]).astype(np.float32)
    got = oracle.e4m3_encode(x)
    ref = torch.from_numpy(x).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    bad = np.nonzero(got != ref)[0]
    assert bad.size == 0, f"{bad.size} codes differ, first x = {x[bad[0]]!r}: {got[bad[0]]:#x} vs {ref[bad[0]]:#x}"


def test_e4m3_encode_saturates_and_keeps_nan():
    x = np.array([464.0, 480.0, 1e6, np.inf, -464.0, -1e9, -np.inf, np.nan], np.float32)
    got = oracle.e4m3_encode(x)
    np.testing.assert_array_equal(got[:4], 0x7E)
    np.testing.assert_array_equal(got[4:7], 0xFE)
    assert np.isnan(oracle.e4m3_decode(got[7:]))[0]


def test_quantize_kv_blocks_scale_bound_and_exact_values():
    """Per (block, head): the largest magnitude maps to 448; every element is within half a code step
    of its value (relative 2^-4 for normal codes, 2^-10 * scale below the normal range); a block
    whose values are already codes times a power-of-two scale comes back exactly; a zero block
    gets scale 0 (no nonzero value yet) and codes 0."""
    rng = np.random.default_rng(1)
    x = rng.standard_normal((6, 2, 16, 128)).astype(np.float32) * rng.uniform(0.01, 50, (6, 2, 1, 1)).astype(np.float32)
    x[5, 1] = 0.0
    codes, scales = oracle.quantize_kv_blocks(x)
    deq = oracle.dequantize_kv_blocks(codes, scales)
    for b in range(6):
        for h in range(2):
            blk, s = x[b, h].astype(np.float64), float(scales[b, h])
            if b == 5 and h == 1:
                assert s == 0.0 and not codes[b, h].any()
                continue
            assert np.isclose(s, np.float32(np.abs(x[b, h]).max() / np.float32(448.0)), rtol=0, atol=0)
            assert np.abs(oracle.e4m3_decode(codes[b, h])).max() == 448.0
            y = np.abs(blk) / s
            bound = np.where(y >= 2.0 ** -6, 2.0 ** -4 * y, 2.0 ** -10) * s * (1 + 1e-6)
            assert np.all(np.abs(deq[b, h] - blk) <= bound + 1e-30)
    # exact round trip: values that are codes times a power-of-two scale with the largest code present
    c = rng.integers(0, 0x7E, (1, 1, 16, 128)).astype(np.uint8)
    c[0, 0, 0, 0] = 0x7E
    exact = (oracle.e4m3_decode(c) * 2.0 ** -3).astype(np.float32)
    codes2, scales2 = oracle.quantize_kv_blocks(exact)
    assert scales2[0, 0] == np.float32(2.0 ** -3)
    np.testing.assert_array_equal(oracle.dequantize_kv_blocks(codes2, scales2), exact.astype(np.float64))


# ------------------------------------------------------------------------------------------------
# FP8 (E4M3) cache written row by row (a decoding loop's append)
# ------------------------------------------------------------------------------------------------

def _rows_into_block(rows, bs=16):
    """slots 0 .. n-1 of block 0 and the rows as [n][Hkv][d]"""
    return np.arange(len(rows), dtype=np.int32), np.ascontiguousarray(rows, np.float32)


def test_append_rows_equal_whole_block_quantization_when_the_first_row_holds_the_max():
    # the scale never grows after row 0, so no row is re-encoded: every row's codes are those of
    # the whole block quantized at once (itself pinned against torch's float8_e4m3fn)
    rng = np.random.default_rng(3)
    x = rng.standard_normal((1, 2, 16, 64)).astype(np.float32)
    x[0, :, 0, 5] = 9.0          # row 0 of each head holds the block's largest magnitude
    x[0, 1, 0, 7] = -11.0
    want_c, want_s = oracle.quantize_kv_blocks(x)
    c0 = np.zeros_like(want_c)
    s0 = np.zeros_like(want_s)
    slots, rows = _rows_into_block(x[0].transpose(1, 0, 2))
    got_c, got_s = oracle.append_kv_quantized(c0, s0, slots, rows)
    np.testing.assert_array_equal(got_s, want_s)
    np.testing.assert_array_equal(got_c, want_c)


def test_append_scale_is_amax_over_rows_so_far_and_power_of_two_growth_is_exact():
    # rows 0..3 each double the block's largest magnitude (scales 2^-2 .. 2^1, exact in fp32), with
    # every value a normal code times its row's scale, at least 2^-2 of a unit: every re-encoding
    # divides by exactly 2 and stays in the normal range, so after all appends the dequantized block
    # is the written rows exactly; the scale after row r is amax(rows <= r) / 448 (the whole-block
    # quantizer's scale of the block truncated to those rows).
    rng = np.random.default_rng(4)
    d = 32
    normal = oracle.e4m3_decode(np.arange(0x28, 0x7F, dtype=np.uint8))      # codes 0.25 .. 448
    rows = np.zeros((16, 1, d), np.float32)
    for r in range(16):
        s_r = 2.0 ** (min(r, 3) - 2)
        vals = rng.choice(normal[normal <= 448.0 / (2.0 if r > 3 else 1.0)], size=d) * rng.choice([-1, 1], size=d)
        vals[rng.integers(0, d)] = 0.0
        if r <= 3:
            vals[0] = 448.0
        rows[r, 0] = (vals * s_r).astype(np.float32)
    c = np.zeros((1, 1, 16, d), np.uint8)
    s = np.zeros((1, 1), np.float32)
    for r in range(16):
        c, s = oracle.append_kv_quantized(c, s, [r], rows[r:r + 1])
        trunc = np.zeros((1, 1, 16, d), np.float32)
        trunc[0, 0, :r + 1] = rows[:r + 1, 0]
        assert s[0, 0] == oracle.quantize_kv_blocks(trunc)[1][0, 0]
    assert s[0, 0] == 2.0
    np.testing.assert_array_equal(oracle.dequantize_kv_blocks(c, s)[0, 0], rows[:, 0].astype(np.float64))


def test_append_re_encoding_stays_within_the_accumulated_rounding_bound():
    # each re-encoding moves a value by at most half a code step at the new scale (relative 2^-4 in
    # the normal range, 2^-10 * scale below it) plus fp32 roundings; a row re-encoded k times is
    # within k + 1 such steps of its value at the final scale
    rng = np.random.default_rng(5)
    d = 128
    rows = (rng.standard_normal((16, 2, d)) * np.exp(rng.uniform(-2, 2, (16, 2, 1)))).astype(np.float32)
    c = np.zeros((1, 2, 16, d), np.uint8)
    s = np.zeros((1, 2), np.float32)
    grown = np.zeros((16, 2), np.int64)
    for r in range(16):
        s_before = s.copy()
        c, s = oracle.append_kv_quantized(c, s, [r], rows[r:r + 1])
        for g in range(2):
            if r > 0 and s[0, g] > s_before[0, g]:
                grown[:r, g] += 1
    deq = oracle.dequantize_kv_blocks(c, s)
    for g in range(2):
        sf = float(s[0, g])
        x = rows[:, g].astype(np.float64)
        step = np.where(np.abs(x) >= 2.0 ** -6 * sf, 2.0 ** -4 * np.abs(x) * 1.07, 2.0 ** -10 * sf)
        bound = (grown[:, g, None] + 1) * step + 1e-7 * sf
        assert np.all(np.abs(deq[0, g] - x) <= bound)
        assert sf == np.float32(np.abs(rows[:, g]).max()) / np.float32(448.0)


def test_append_row_zero_starts_a_reused_block_afresh_and_zero_rows_keep_scale_zero():
    rng = np.random.default_rng(6)
    d = 16
    # a block handed out again: stale codes and scale from a former owner
    c = rng.integers(0, 0x7E, (2, 1, 16, d)).astype(np.uint8)
    s = np.array([[3.5], [0.25]], np.float32)
    x = rng.standard_normal((1, 1, d)).astype(np.float32)
    c2, s2 = oracle.append_kv_quantized(c, s, [16], x)          # block 1, row 0
    assert s2[1, 0] == np.float32(np.abs(x).max()) / np.float32(448.0)
    np.testing.assert_array_equal(c2[1, 0, 1:], c[1, 0, 1:])    # later rows untouched
    np.testing.assert_array_equal(c2[0], c[0])                  # other blocks untouched
    ref = torch.from_numpy(x[0, 0] / s2[1, 0]).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    np.testing.assert_array_equal(c2[1, 0, 0], ref)
    # zero rows: the scale stays 0 and the codes 0 until a nonzero row arrives, which does not
    # touch them
    c = np.zeros((1, 1, 16, d), np.uint8)
    s = np.zeros((1, 1), np.float32)
    c, s = oracle.append_kv_quantized(c, s, [0, 1, 2], np.zeros((3, 1, d), np.float32))
    assert s[0, 0] == 0.0 and not c.any()
    c, s = oracle.append_kv_quantized(c, s, [3], x)
    assert s[0, 0] == np.float32(np.abs(x).max()) / np.float32(448.0) and not c[0, 0, :3].any()


def test_decode_f64_and_paged_decode_equal_the_fp32_row_decode():
    # the fp64-row decode is the same arithmetic as oracle.decode on fp32-exact rows, and the paged
    # form, which gathers each stream's rows through the block tables, reads exactly those rows
    from paper_2608_06146_gb300 import inputs
    pages = [inputs.PageSpec(40, 9, [0, 9, 4], [3, 20, 17]), inputs.PageSpec(5, 16, [16, 2], [1, 33])]
    wl = inputs.Workload("pin", pages, 8, 2, 16, torch.bfloat16, "decode")
    di = inputs.decode_inputs(wl, 9, layout_streams=True)
    o32, l32 = oracle.decode_pages(pages, di, 0.3, layout_streams=True)
    sp, sh, pl = oracle.decode_streams(pages, layout_streams=True)
    f64 = lambda t: t.double().numpy()
    o64, l64 = oracle.decode_f64(sp, sh, pl, di.page_off, di.priv_off, f64(di.stream_k), f64(di.stream_v),
                                 f64(di.priv_k), f64(di.priv_v), di.q, 0.3)
    np.testing.assert_array_equal(o64, o32)
    np.testing.assert_array_equal(l64, l32)
    op, lp = oracle.decode_paged(pages, di.k_pool, di.v_pool, di.page_table, di.stream_table, di.q, 0.3,
                                 layout_streams=True)
    np.testing.assert_array_equal(op, o32)
    np.testing.assert_array_equal(lp, l32)


def test_prefill_dense_rows_is_the_dense_prefill_on_those_rows():
    # the row-selected form reads the same visibility and does the same arithmetic per row, so its
    # rows are bit-identical to the full function's (itself pinned above)
    pages = [(13, 9, [3, 9, 0], [4, 6, 2]), (0, 5, [5, 1], [3, 7]), (20, 0, [0], [5])]
    T = oracle.total_tokens(pages)
    q, k, v = _qkv(T, 4, 2, 8, seed=21)
    o_all, l_all = oracle.prefill_dense(pages, q, k, v, 0.3)
    rows = np.array([0, 5, 21, 22, 25, 33, T - 1, 40, 41], np.int64)
    o, l = oracle.prefill_dense_rows(pages, q[rows], k, v, 0.3, rows)
    np.testing.assert_array_equal(o, o_all[rows])
    np.testing.assert_array_equal(l, l_all[rows])
