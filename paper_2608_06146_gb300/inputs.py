"""Seeded synthetic workloads for ancestor-masked attention.

This module only draws page structures and random tensors and lays a logical KV cache out in
paged blocks. It holds none of the attention arithmetic, so both the CUDA path and the CPU oracle
can be fed from it.

Shapes follow the paper's setting: a Qwen3-VL-2B-style decoder with 16 query heads, 2 KV heads
and head_dim 128, and a bf16 KV cache in 16-token blocks (Sec. 4 serving setup; App. E.2). The
paper's page data is not reproduced: page sizes, branch counts and lengths are drawn from the
distributions stated for each workload below.

Every random draw uses numpy ``default_rng(seed)`` for integers and a seeded ``torch.Generator``
(CPU) for tensor values.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np
import torch


@dataclass
class PageSpec:
    """One page: prefix X of ``prefix_len`` tokens, a layout stream of ``layout_len`` tokens and
    ``len(branch_len)`` content branches. ``fork_offset[k]`` is the number of layout-stream tokens
    branch k sees; ``branch_len[k]`` is its token count (prefill) or its private KV length
    including the token being decoded (decode)."""

    prefix_len: int
    layout_len: int
    fork_offset: List[int] = field(default_factory=list)
    branch_len: List[int] = field(default_factory=list)

    @property
    def num_branches(self) -> int:
        return len(self.branch_len)

    @property
    def stream_len(self) -> int:
        return self.prefix_len + self.layout_len

    @property
    def packed_len(self) -> int:
        return self.prefix_len + self.layout_len + int(sum(self.branch_len))


@dataclass
class Workload:
    name: str
    pages: List[PageSpec]
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    dtype: torch.dtype
    kind: str  # "decode", "prefill" or "both"
    block_size: int = 16


# --------------------------------------------------------------------------------------------
# Page structures of the five workloads
# --------------------------------------------------------------------------------------------

def tiny_page(seed: int = 0) -> Workload:
    """Bring-up page: prefix 256, layout stream 32 with 4 records at seeded increasing offsets,
    branch lengths {8,16,24,32}, 4 query heads / 1 KV head, head_dim 64, fp32."""
    rng = np.random.default_rng(seed)
    forks = sorted(int(x) for x in rng.choice(np.arange(1, 33), size=4, replace=False))
    page = PageSpec(256, 32, forks, [8, 16, 24, 32])
    return Workload("tiny single page (fp32, P=256 L=32 N=4)", [page], 4, 1, 64, torch.float32, "both")


def decode_page(seed: int = 1) -> Workload:
    """One page, decode step: prefix 2048 (1792 visual + 256 prompt), layout stream 256, 16 branches
    with private KV lengths uniform in [16,256], 16 q heads / 2 KV heads, head_dim 128, bf16."""
    rng = np.random.default_rng(seed)
    forks = sorted(int(x) for x in rng.choice(np.arange(1, 257), size=16, replace=False))
    lens = [int(x) for x in rng.integers(16, 257, size=16)]
    return Workload("one page decode (P=2048 L=256 N=16)", [PageSpec(2048, 256, forks, lens)],
                    16, 2, 128, torch.bfloat16, "decode")


def dense_page(seed: int = 2) -> Workload:
    """Table/formula-heavy page, decode step: prefix 4096, layout stream 512, 64 branches with
    log-normal private lengths (median 64, sigma 1.0, capped at 1024)."""
    rng = np.random.default_rng(seed)
    forks = sorted(int(x) for x in rng.choice(np.arange(1, 513), size=64, replace=False))
    z = rng.standard_normal(64)
    lens = [int(x) for x in np.clip(np.round(np.exp(np.log(64.0) + 1.0 * z)), 1, 1024)]
    return Workload("dense page decode (P=4096 L=512 N=64)", [PageSpec(4096, 512, forks, lens)],
                    16, 2, 128, torch.bfloat16, "decode")


def serving_batch(seed: int = 3, num_pages: int = 32) -> Workload:
    """Concurrent serving batch, decode step: 32 pages, prefix uniform in [1024,4096], branches per
    page Poisson(20) clipped to [1,64], 8 layout tokens per record (f_k = 8k), private lengths
    log-normal (median 96, sigma 1.0, cap 2048)."""
    rng = np.random.default_rng(seed)
    pages = []
    for _ in range(num_pages):
        P = int(rng.integers(1024, 4097))
        N = int(np.clip(rng.poisson(20), 1, 64))
        z = rng.standard_normal(N)
        lens = [int(x) for x in np.clip(np.round(np.exp(np.log(96.0) + 1.0 * z)), 1, 2048)]
        pages.append(PageSpec(P, 8 * N, [8 * (k + 1) for k in range(N)], lens))
    return Workload(f"serving batch decode ({num_pages} pages)", pages, 16, 2, 128, torch.bfloat16, "decode")


def packed_prefill(seed: int = 4, num_pages: int = 8, page_tokens: int = 4096,
                   shuffle_branches: bool = False) -> Workload:
    """Packed variable-length ancestor prefill: 8 pages x 4096 tokens = 32768. Per page prefix
    uniform in [1024,3072], N uniform in [8,48], 8 layout tokens per record (f_k = 8k), raw branch
    lengths log-normal (median 80, sigma 0.75) rescaled to fill the page (floor, each >= 1, the
    remainder to the last branch; N shrinks when the budget is below N). ``shuffle_branches``
    permutes the branches of each page so that f_k is not monotone in k."""
    rng = np.random.default_rng(seed)
    pages = []
    for _ in range(num_pages):
        P = int(rng.integers(1024, 3073))
        N = int(rng.integers(8, 49))
        L = 8 * N
        budget = page_tokens - P - L
        if budget < N:
            N = max(budget // 9, 0)
            L = 8 * N
            budget = page_tokens - P - L
        z = rng.standard_normal(N)
        raw = np.exp(np.log(80.0) + 0.75 * z)
        lens = np.maximum(np.floor(raw * budget / raw.sum()).astype(np.int64), 1)
        while lens.sum() > budget:  # the floor of >= 1 can overshoot a tight budget
            lens[int(np.argmax(lens))] -= 1
        lens[-1] += budget - int(lens.sum())
        forks = [8 * (k + 1) for k in range(N)]
        lens = [int(x) for x in lens]
        if shuffle_branches and N > 1:
            perm = rng.permutation(N)
            forks = [forks[i] for i in perm]
            lens = [lens[i] for i in perm]
        if N == 0:  # a page with no room for branches becomes one causal stream
            P = page_tokens
        pages.append(PageSpec(P, L, forks, lens))
    return Workload(f"packed prefill ({num_pages} pages x {page_tokens} tokens)", pages, 16, 2, 128,
                    torch.bfloat16, "prefill")


WORKLOADS = {
    "tiny": tiny_page,
    "decode_page": decode_page,
    "dense_page": dense_page,
    "serving_batch": serving_batch,
    "packed_prefill": packed_prefill,
}


# --------------------------------------------------------------------------------------------
# A synthetic token source for the decoding loop (Algorithm 1)
# --------------------------------------------------------------------------------------------

class LoopTokenSource:
    """Stands in for the decoder inside Algorithm 1's loop over ``pages``: each output's event comes
    from the page structure alone, never from the attention outputs. The layout stream of a page
    completes region B_k (a fork) when its c-th token is in the cache and f_k = c, and outputs EOS
    after its L-th token; branch k outputs EOS after its n_k-th token; branches with f_k = 0 fork
    from the prefill's output. Every input's Q/K/V is the row of the packed tensors (pages back to
    back, each [X | layout | Y_1 | ... | Y_N], as ``packed_qkv`` draws them) of the token it is, so a
    loop run decodes exactly the tokens of the packed pages.

    Stream ids are the scheduler's; the source learns them from ``admitted`` and ``forked``.
    Per-stream state is kept in arrays indexed by stream id, so a step costs a few numpy calls."""

    def __init__(self, pages: Sequence[PageSpec]):
        self.pages = list(pages)
        n = len(self.pages)
        lens = [pg.packed_len for pg in self.pages]
        self.base = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int64) if lens else np.zeros(0, np.int64)
        self.ybase = [[pg.prefix_len + pg.layout_len + int(sum(pg.branch_len[:k])) for k in range(pg.num_branches)]
                      for pg in self.pages]
        self._P = np.asarray([pg.prefix_len for pg in self.pages], np.int64)
        self._L = np.asarray([pg.layout_len for pg in self.pages], np.int64)
        nb = [pg.num_branches for pg in self.pages]
        self._kbase = np.concatenate([[0], np.cumsum(nb)[:-1]]).astype(np.int64) if n else np.zeros(0, np.int64)
        # one unused element at the end: np.where evaluates both of its arms, so a layout stream's
        # lookup of these per-branch arrays needs an index even when no page has a branch
        self._yabs = np.asarray([self.base[p] + y for p in range(n) for y in self.ybase[p]] + [0], np.int64)
        self._nlen = np.asarray([x for pg in self.pages for x in pg.branch_len] + [0], np.int64)
        self._forks_by_count = []
        for pg in self.pages:
            d = {}
            for k, f in enumerate(pg.fork_offset):
                d.setdefault(int(f), []).append(k)
            self._forks_by_count.append(d)
        # forks per (page, layout tokens in the cache), flattened: page p's counts c = 0..L start at _fbase[p]
        self._fbase = np.concatenate([[0], np.cumsum([pg.layout_len + 1 for pg in self.pages])[:-1]]).astype(np.int64) \
            if n else np.zeros(0, np.int64)
        self._fcount = np.zeros(int(sum(pg.layout_len + 1 for pg in self.pages)) + 1, np.int32)
        for p, pg in enumerate(self.pages):
            for f in pg.fork_offset:
                self._fcount[self._fbase[p] + int(f)] += 1
        cap = n + int(sum(nb))           # every stream ever: one layout stream and N branches per page
        self._page = np.full(max(cap, 1), -1, np.int64)
        self._flat = np.full(max(cap, 1), -1, np.int64)   # -1: layout stream, else flat branch index
        self._count = np.zeros(max(cap, 1), np.int64)
        self._pending = {}

    def _grow(self, sid: int) -> None:
        if sid >= self._page.size:
            extra = sid + 1 - self._page.size
            self._page = np.concatenate([self._page, np.full(extra, -1, np.int64)])
            self._flat = np.concatenate([self._flat, np.full(extra, -1, np.int64)])
            self._count = np.concatenate([self._count, np.zeros(extra, np.int64)])

    def _set(self, sid: int, p: int, k: int) -> None:
        self._grow(sid)
        self._page[sid] = p
        self._flat[sid] = -1 if k < 0 else self._kbase[p] + k
        self._count[sid] = 0

    def _forks_at(self, p: int, c: int) -> List[int]:
        return self._forks_by_count[p].get(int(c), [])

    def stream_of(self, sid: int):
        """(page, branch index or -1 for the layout stream) of a stream."""
        p = int(self._page[sid])
        f = int(self._flat[sid])
        return p, (-1 if f < 0 else f - int(self._kbase[p]))

    def admission(self, p: int):
        """(prefix_len, num_forks, layout_eos, prefix rows int64 [P]) of page p's prefill output."""
        pg = self.pages[p]
        rows = self.base[p] + np.arange(pg.prefix_len, dtype=np.int64)
        return pg.prefix_len, len(self._forks_at(p, 0)), pg.layout_len == 0, rows

    def admitted(self, p: int, new_streams) -> None:
        if int(new_streams[0]) >= 0:
            self._set(int(new_streams[0]), p, -1)
        for sid, k in zip(new_streams[1:], self._forks_at(p, 0)):
            self._set(int(sid), p, k)

    def rows(self, ids) -> np.ndarray:
        """Packed rows of the inputs the given streams append now (each stream's next token)."""
        ids = np.asarray(ids, np.int64)
        pg, fl, c = self._page[ids], self._flat[ids], self._count[ids]
        lay = fl < 0
        out = np.where(lay, self.base[pg] + self._P[pg] + c, self._yabs[np.where(lay, 0, fl)] + c)
        self._count[ids] = c + 1
        return out

    def peek_rows(self, ids) -> np.ndarray:
        """rows(ids) without advancing: each stream's next input row (meaningless for a stream that is
        not live)."""
        ids = np.asarray(ids, np.int64)
        pg, fl, c = self._page[ids], self._flat[ids], self._count[ids]
        lay = fl < 0
        return np.where(lay, self.base[pg] + self._P[pg] + c, self._yabs[np.where(lay, 0, fl)] + c)

    def events(self, ids):
        """(num_forks int32 [C], eos uint8 [C]) of the outputs of this step's streams."""
        ids = np.asarray(ids, np.int64)
        pg, fl, c = self._page[ids], self._flat[ids], self._count[ids]
        lay = fl < 0
        eos = np.where(lay, c == self._L[pg], c == self._nlen[np.where(lay, 0, fl)]).astype(np.uint8)
        nf = np.where(lay, self._fcount[np.where(lay, self._fbase[pg] + np.minimum(c, self._L[pg]), 0)], 0).astype(np.int32)
        for i in np.nonzero(nf)[0]:
            self._pending[int(ids[i])] = self._forks_at(int(pg[i]), int(c[i]))
        return nf, eos

    def forked(self, ids, num_forks, new_streams) -> None:
        """Records the ids the scheduler gave the branches forked at this step (in step order)."""
        j = 0
        for i in np.nonzero(np.asarray(num_forks))[0]:
            sid = int(ids[i])
            p = int(self._page[sid])
            for k in self._pending.pop(sid):
                self._set(int(new_streams[j]), p, k)
                j += 1

    def token_rows(self, ids) -> np.ndarray:
        """Packed rows of the tokens the given streams appended last."""
        ids = np.asarray(ids, np.int64)
        pg, fl, c = self._page[ids], self._flat[ids], self._count[ids]
        lay = fl < 0
        return np.where(lay, self.base[pg] + self._P[pg] + c - 1, self._yabs[np.where(lay, 0, fl)] + c - 1)

    def token_row(self, sid: int) -> int:
        return int(self.token_rows([sid])[0])


# --------------------------------------------------------------------------------------------
# Tensors
# --------------------------------------------------------------------------------------------

def randn(shape: Sequence[int], dtype: torch.dtype, seed: int, scale: float = 1.0) -> torch.Tensor:
    """Seeded N(0, scale^2) values on the CPU, rounded once to ``dtype``."""
    g = torch.Generator().manual_seed(int(seed))
    x = torch.randn(*shape, generator=g, dtype=torch.float32)
    if scale != 1.0:
        x = x * scale
    return x.to(dtype)


def packed_qkv(wl: Workload, seed: int, scale: float = 1.0):
    """Packed Q [T][Hq][d] and K, V [T][Hkv][d] in ``wl.dtype`` on the CPU."""
    T = sum(p.packed_len for p in wl.pages)
    q = randn((T, wl.num_q_heads, wl.head_dim), wl.dtype, seed * 1000 + 1, scale)
    k = randn((T, wl.num_kv_heads, wl.head_dim), wl.dtype, seed * 1000 + 2, scale)
    v = randn((T, wl.num_kv_heads, wl.head_dim), wl.dtype, seed * 1000 + 3, scale)
    return q, k, v


def packed_dout(wl: Workload, seed: int, scale: float = 1.0) -> torch.Tensor:
    """Upstream gradient dO [T][Hq][d] of a packed prefill, in ``wl.dtype`` on the CPU."""
    T = sum(p.packed_len for p in wl.pages)
    return randn((T, wl.num_q_heads, wl.head_dim), wl.dtype, seed * 1000 + 4, scale)


@dataclass
class DecodeInputs:
    """Logical (unpaged) decode-step state plus its paged layout.

    Streams are page-major, branches in page order, then (if ``layout_streams``) the page's layout
    stream last. ``stream_k/v``: every page's shared stream rows back to back, [rows][Hkv][d];
    ``priv_k/v``: every stream's private rows back to back. ``k_pool``/``v_pool``:
    [num_blocks][Hkv][block][d]; ``page_table``: [pages][page_stride] block ids of the shared
    stream; ``stream_table``: [streams][stream_stride] block ids of the private rows."""

    q: torch.Tensor
    stream_k: torch.Tensor
    stream_v: torch.Tensor
    priv_k: torch.Tensor
    priv_v: torch.Tensor
    page_off: np.ndarray
    priv_off: np.ndarray
    stream_page: np.ndarray
    priv_len: np.ndarray
    k_pool: torch.Tensor
    v_pool: torch.Tensor
    page_table: np.ndarray
    stream_table: np.ndarray
    num_blocks: int


def decode_stream_order(wl: Workload, layout_streams: bool = False):
    """(stream_page, priv_len) in the stream order described in ``DecodeInputs``: each page's
    branches with their private lengths as drawn, then (with ``layout_streams``) its layout stream,
    which has no private rows. Where each stream's view of the shared stream ends is not decided
    here."""
    sp, pl = [], []
    for p, pg in enumerate(wl.pages):
        for n in pg.branch_len:
            sp.append(p); pl.append(n)
        if layout_streams:
            sp.append(p); pl.append(0)
    return np.asarray(sp, np.int32), np.asarray(pl, np.int32)


def decode_inputs(wl: Workload, seed: int, layout_streams: bool = False, scale: float = 1.0,
                  pool_slack: float = 2.0, q_override: Optional[torch.Tensor] = None) -> DecodeInputs:
    """Random logical cache and queries for one decode step, scattered into a block pool whose
    block ids are a seeded random permutation (the pool holds ``pool_slack`` x the needed blocks)."""
    bs, Hkv, d, Hq = wl.block_size, wl.num_kv_heads, wl.head_dim, wl.num_q_heads
    stream_page, priv_len = decode_stream_order(wl, layout_streams)
    S = len(stream_page)
    page_rows = np.asarray([pg.stream_len for pg in wl.pages], np.int64)
    page_off = np.concatenate([[0], np.cumsum(page_rows)[:-1]]).astype(np.int64)
    priv_off = np.concatenate([[0], np.cumsum(priv_len.astype(np.int64))[:-1]]).astype(np.int64) if S else np.zeros(0, np.int64)
    n_stream_rows = int(page_rows.sum())
    n_priv_rows = int(priv_len.astype(np.int64).sum())
    stream_k = randn((n_stream_rows, Hkv, d), wl.dtype, seed * 1000 + 11, scale)
    stream_v = randn((n_stream_rows, Hkv, d), wl.dtype, seed * 1000 + 12, scale)
    priv_k = randn((n_priv_rows, Hkv, d), wl.dtype, seed * 1000 + 13, scale)
    priv_v = randn((n_priv_rows, Hkv, d), wl.dtype, seed * 1000 + 14, scale)
    q = q_override if q_override is not None else randn((S, Hq, d), wl.dtype, seed * 1000 + 15, scale)

    page_blocks = [(int(r) + bs - 1) // bs for r in page_rows]
    priv_blocks = [(int(r) + bs - 1) // bs for r in priv_len]
    need = sum(page_blocks) + sum(priv_blocks)
    num_blocks = max(int(need * pool_slack), need, 1)
    rng = np.random.default_rng(seed * 7919 + 17)
    perm = rng.permutation(num_blocks)
    page_stride = max(max(page_blocks, default=0), 1)
    stream_stride = max(max(priv_blocks, default=0), 1)
    page_table = np.full((len(wl.pages), page_stride), -1, np.int32)
    stream_table = np.full((S, stream_stride), -1, np.int32)
    k_pool = torch.zeros((num_blocks, Hkv, bs, d), dtype=wl.dtype)
    v_pool = torch.zeros((num_blocks, Hkv, bs, d), dtype=wl.dtype)
    nxt = 0

    def scatter(rows_k, rows_v, n_rows, table_row):
        nonlocal nxt
        for b in range((n_rows + bs - 1) // bs):
            blk = int(perm[nxt]); nxt += 1
            table_row[b] = blk
            lo, hi = b * bs, min(n_rows, (b + 1) * bs)
            k_pool[blk, :, : hi - lo, :] = rows_k[lo:hi].transpose(0, 1)
            v_pool[blk, :, : hi - lo, :] = rows_v[lo:hi].transpose(0, 1)

    for p in range(len(wl.pages)):
        lo = int(page_off[p]); n = int(page_rows[p])
        scatter(stream_k[lo:lo + n], stream_v[lo:lo + n], n, page_table[p])
    for s in range(S):
        lo = int(priv_off[s]); n = int(priv_len[s])
        scatter(priv_k[lo:lo + n], priv_v[lo:lo + n], n, stream_table[s])
    return DecodeInputs(q, stream_k, stream_v, priv_k, priv_v, page_off, priv_off, stream_page,
                        priv_len, k_pool, v_pool, page_table, stream_table, num_blocks)
