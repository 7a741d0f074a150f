"""fp64 CPU oracle for PaDoc ancestor-masked attention (ctypes wrapper of padoc_oracle.c).

TEST INFRASTRUCTURE ONLY: tests/, ``__graft_entry__.smoke()`` and bench.py's cpu_baseline and
reference legs may use it; the product path never does. It imports nothing from the CUDA
package. Pages are given as objects with ``prefix_len``, ``layout_len``, ``fork_offset`` and
``branch_len`` (or as ``(P, L, forks, lens)`` tuples).

Every function follows the paper's definition of the visibility (Sec. 3.2 ancestor sets;
App. C.1 packed statement; App. E.1 additive-bias softmax and Algorithm 1); the C source states
the readings taken where the paper is silent. Parity of all functions is pinned by
tests/test_oracle_pins.py against closed forms, torch's SDPA, a simulator of Algorithm 1's mask
recurrence and hand-derived fixtures; the backward against central differences of the forward,
torch autograd through the per-branch gather, and closed forms. The FP8 (E4M3) KV-cache
definitions (encode, decode, per-block quantization) are pinned against torch's float8_e4m3fn on
every code and on every tie between neighbouring codes, and by the format's error bound.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "padoc_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_build", "libpadoc_oracle.so")
_lib = None
_lock = threading.Lock()

_i32p = ctypes.POINTER(ctypes.c_int32)
_i64p = ctypes.POINTER(ctypes.c_int64)
_f32p = ctypes.POINTER(ctypes.c_float)
_f64p = ctypes.POINTER(ctypes.c_double)
_u8p = ctypes.POINTER(ctypes.c_uint8)
_i8p = ctypes.POINTER(ctypes.c_int8)


def build(force: bool = False) -> str:
    """Compile padoc_oracle.c with gcc (fp64, OpenMP) into oracle/_build/."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.oracle_total_tokens.restype = ctypes.c_int64
            lib.oracle_total_tokens.argtypes = [_i32p, ctypes.c_int32, _i32p]
            lib.oracle_dense_mask.argtypes = [_i32p, ctypes.c_int32, _i32p, _i32p, ctypes.c_int32, _u8p]
            lib.oracle_spans.argtypes = [_i32p, ctypes.c_int32, _i32p, _i32p, _i32p]
            pre = [_i32p, ctypes.c_int32, _i32p, _i32p, _f32p, _f32p, _f32p, ctypes.c_int32,
                   ctypes.c_int32, ctypes.c_int32, ctypes.c_double, _f64p, _f64p]
            lib.oracle_prefill_dense.argtypes = pre
            lib.oracle_prefill_gather.argtypes = pre
            lib.oracle_decode.argtypes = [ctypes.c_int32, _i32p, _i32p, _i32p, _i64p, _i64p, _f32p, _f32p,
                                          _f32p, _f32p, _f32p, ctypes.c_int32, ctypes.c_int32,
                                          ctypes.c_int32, ctypes.c_double, _f64p, _f64p]
            lib.oracle_merge.argtypes = [_f64p, _f64p, ctypes.c_int32, ctypes.c_int64, ctypes.c_int32,
                                         _f64p, _f64p]
            lib.oracle_tile_kinds.argtypes = [_i32p, ctypes.c_int32, _i32p, _i32p, ctypes.c_int32,
                                              ctypes.c_int32, _i8p]
            lib.oracle_prefill_bwd.argtypes = [_i32p, ctypes.c_int32, _i32p, _i32p, _f32p, _f32p, _f32p,
                                               _f32p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                               ctypes.c_double, ctypes.c_int64, _i64p, ctypes.c_int64,
                                               _i64p, _f64p, _f64p, _f64p]
            lib.oracle_e4m3_encode.argtypes = [_f32p, ctypes.c_int64, _u8p]
            lib.oracle_e4m3_decode.argtypes = [_u8p, ctypes.c_int64, _f64p]
            lib.oracle_quantize_kv_blocks.argtypes = [_f32p, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                                      ctypes.c_int32, _u8p, _f32p]
            lib.oracle_dequantize_kv_blocks.argtypes = [_u8p, _f32p, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                                        ctypes.c_int32, _f64p]
            lib.oracle_prefill_dense_rows.argtypes = [_i32p, ctypes.c_int32, _i32p, _i32p, _f32p, _f32p, _f32p,
                                                      ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_double,
                                                      ctypes.c_int64, _i64p, _f64p, _f64p]
            lib.oracle_append_kv_quantized.argtypes = [_u8p, _f32p, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                                       ctypes.c_int32, _i32p, ctypes.c_int32, _f32p]
            lib.oracle_decode_f64.argtypes = [ctypes.c_int32, _i32p, _i32p, _i32p, _i64p, _i64p, _f64p, _f64p,
                                              _f64p, _f64p, _f32p, ctypes.c_int32, ctypes.c_int32,
                                              ctypes.c_int32, ctypes.c_double, _f64p, _f64p]
            _lib = lib
    return _lib


def _ptr(a, t):
    return a.ctypes.data_as(t)


def _flat(pages):
    pln, forks, lens = [], [], []
    for pg in pages:
        if isinstance(pg, tuple):
            P, L, f, n = pg
        else:
            P, L, f, n = pg.prefix_len, pg.layout_len, pg.fork_offset, pg.branch_len
        assert len(f) == len(n)
        pln += [int(P), int(L), len(n)]
        forks += [int(x) for x in f]
        lens += [int(x) for x in n]
    z = lambda x: np.ascontiguousarray(np.asarray(x if x else [0], np.int32))
    return z(pln), len(pages), z(forks), z(lens)


def _f32(x):
    """Exact fp32 copy of a torch tensor or array (bf16 and fp32 convert exactly)."""
    try:
        import torch
        if isinstance(x, torch.Tensor):
            return np.ascontiguousarray(x.detach().to("cpu", torch.float32).numpy())
    except ImportError:  # pragma: no cover
        pass
    return np.ascontiguousarray(np.asarray(x, np.float32))


def total_tokens(pages) -> int:
    pln, n, f, b = _flat(pages)
    return int(_load().oracle_total_tokens(_ptr(pln, _i32p), n, _ptr(b, _i32p)))


def dense_mask(pages, page: int) -> np.ndarray:
    """[S_p][S_p] visibility (uint8) of one page, from node membership and ancestor sets."""
    pln, n, f, b = _flat(pages)
    pg = pages[page]
    S = pg[0] + pg[1] + sum(pg[3]) if isinstance(pg, tuple) else pg.prefix_len + pg.layout_len + sum(pg.branch_len)
    m = np.zeros((S, S), np.uint8)
    _load().oracle_dense_mask(_ptr(pln, _i32p), n, _ptr(f, _i32p), _ptr(b, _i32p), page, _ptr(m, _u8p))
    return m


def spans(pages) -> np.ndarray:
    """[T][4] int32 visible spans {kv0_begin, kv0_end, kv1_begin, kv1_end} (absolute packed)."""
    pln, n, f, b = _flat(pages)
    T = total_tokens(pages)
    out = np.zeros((max(T, 1), 4), np.int32)
    _load().oracle_spans(_ptr(pln, _i32p), n, _ptr(f, _i32p), _ptr(b, _i32p), _ptr(out, _i32p))
    return out[:T]


def _prefill(fn_name, pages, q, k, v, scale):
    pln, n, f, b = _flat(pages)
    q, k, v = _f32(q), _f32(k), _f32(v)
    T, Hq, d = q.shape
    Hkv = k.shape[1]
    assert k.shape == (T, Hkv, d) and v.shape == (T, Hkv, d) and Hq % Hkv == 0
    o = np.zeros((T, Hq, d), np.float64)
    lse = np.zeros((T, Hq), np.float64)
    getattr(_load(), fn_name)(_ptr(pln, _i32p), n, _ptr(f, _i32p), _ptr(b, _i32p), _ptr(q, _f32p),
                              _ptr(k, _f32p), _ptr(v, _f32p), Hq, Hkv, d, float(scale),
                              _ptr(o, _f64p), _ptr(lse, _f64p))
    return o, lse


def prefill_dense(pages, q, k, v, scale):
    """Packed prefill via the dense ancestor visibility. Returns fp64 (O [T][Hq][d], LSE [T][Hq])."""
    return _prefill("oracle_prefill_dense", pages, q, k, v, scale)


def prefill_dense_rows(pages, q_rows, k, v, scale, rows):
    """``prefill_dense`` on the absolute packed rows ``rows`` only: q_rows [n][Hq][d] are those rows'
    queries, k / v the whole packed [T][Hkv][d]. Returns fp64 (O [n][Hq][d], LSE [n][Hq])."""
    pln, n, f, b = _flat(pages)
    qs, k, v = _f32(q_rows), _f32(k), _f32(v)
    r = np.ascontiguousarray(np.asarray(rows, np.int64))
    T = total_tokens(pages)
    assert k.shape[0] == T and v.shape == k.shape and qs.shape[0] == len(r) and ((r >= 0) & (r < T)).all()
    Hq, d = qs.shape[1], qs.shape[2]
    o = np.zeros((len(r), Hq, d), np.float64)
    lse = np.zeros((len(r), Hq), np.float64)
    if len(r):
        _load().oracle_prefill_dense_rows(_ptr(pln, _i32p), n, _ptr(f, _i32p), _ptr(b, _i32p), _ptr(qs, _f32p),
                                          _ptr(k, _f32p), _ptr(v, _f32p), Hq, k.shape[1], d, float(scale), len(r),
                                          _ptr(r, _i64p), _ptr(o, _f64p), _ptr(lse, _f64p))
    return o, lse


def prefill_gather(pages, q, k, v, scale):
    """Packed prefill via per-branch gather and bottom-right causal attention."""
    return _prefill("oracle_prefill_gather", pages, q, k, v, scale)


def decode_streams(pages, layout_streams: bool = False):
    """The per-stream decode plan {page, shared_len, private_len} of a decode step, in stream order
    (each page's branches in order, then with ``layout_streams`` its layout stream).

    Sec. 3.2 gives branch k the ancestors {X, B_<=k}: the whole prefix X and the layout-stream
    tokens written before it forked, f_k of them (Algorithm 1 copies the layout row before the
    region's boundary output is appended), so its cutoff on the page's shared stream [X | layout]
    is P + f_k and its private rows are its own n_k tokens, the newest being the one decoded
    (Algorithm 1 appends before it decodes). The layout stream sees the prefix and all L of its own
    tokens and has no private rows: cutoff P + L, private 0."""
    sp, sh, pl = [], [], []
    for p, pg in enumerate(pages):
        if isinstance(pg, tuple):
            P, L, forks, lens = pg
        else:
            P, L, forks, lens = pg.prefix_len, pg.layout_len, pg.fork_offset, pg.branch_len
        for f, n in zip(forks, lens):
            assert 0 <= f <= L and n >= 1
            sp.append(p); sh.append(P + f); pl.append(n)
        if layout_streams:
            sp.append(p); sh.append(P + L); pl.append(0)
    return np.asarray(sp, np.int32), np.asarray(sh, np.int32), np.asarray(pl, np.int32)


def decode_pages(pages, di, scale, layout_streams: bool = False):
    """``decode`` of every stream of ``pages`` over the logical rows of ``di`` (an object with the
    fields page_off, priv_off, stream_k, stream_v, priv_k, priv_v and q laid out as the seeded
    input generator does), each stream's cutoff and private length taken from ``decode_streams``."""
    sp, sh, pl = decode_streams(pages, layout_streams)
    assert np.array_equal(sp, np.asarray(di.stream_page)) and np.array_equal(pl, np.asarray(di.priv_len))
    return decode(sp, sh, pl, di.page_off, di.priv_off, di.stream_k, di.stream_v, di.priv_k, di.priv_v, di.q, scale)


def decode(stream_page, shared_len, priv_len, page_off, priv_off, stream_k, stream_v, priv_k, priv_v,
           q, scale):
    """One decode step over logical (unpaged) K/V; see padoc_oracle.c:oracle_decode."""
    sp = np.ascontiguousarray(np.asarray(stream_page, np.int32))
    sh = np.ascontiguousarray(np.asarray(shared_len, np.int32))
    pl = np.ascontiguousarray(np.asarray(priv_len, np.int32))
    po = np.ascontiguousarray(np.asarray(page_off, np.int64))
    vo = np.ascontiguousarray(np.asarray(priv_off, np.int64))
    sk, sv, pk, pv, qq = (_f32(x) for x in (stream_k, stream_v, priv_k, priv_v, q))
    S, Hq, d = qq.shape
    Hkv = sk.shape[1] if sk.size else pk.shape[1]
    guard = lambda a: a if a.size else np.zeros((1, Hkv, d), np.float32)
    sk, sv, pk, pv = guard(sk), guard(sv), guard(pk), guard(pv)
    o = np.zeros((S, Hq, d), np.float64)
    lse = np.zeros((S, Hq), np.float64)
    if S:
        _load().oracle_decode(S, _ptr(sp, _i32p), _ptr(sh, _i32p), _ptr(pl, _i32p), _ptr(po, _i64p),
                              _ptr(vo, _i64p), _ptr(sk, _f32p), _ptr(sv, _f32p), _ptr(pk, _f32p),
                              _ptr(pv, _f32p), _ptr(qq, _f32p), Hq, Hkv, d, float(scale),
                              _ptr(o, _f64p), _ptr(lse, _f64p))
    return o, lse


def merge(part_o, part_lse):
    """Merge partial softmax results over disjoint key sets: part_o [S][rows][d], part_lse [S][rows]."""
    po = np.ascontiguousarray(np.asarray(part_o, np.float64))
    pl = np.ascontiguousarray(np.asarray(part_lse, np.float64))
    S, R, d = po.shape
    o = np.zeros((R, d), np.float64)
    lse = np.zeros((R,), np.float64)
    _load().oracle_merge(_ptr(po, _f64p), _ptr(pl, _f64p), S, R, d, _ptr(o, _f64p), _ptr(lse, _f64p))
    return o, lse


def tile_kinds(pages, q_tile: int, k_tile: int) -> np.ndarray:
    """[q_tiles][k_tiles] int8: 0 no visible pair, 1 PARTIAL, 2 FULL (brute force; small inputs)."""
    pln, n, f, b = _flat(pages)
    T = total_tokens(pages)
    nq, nk = -(-T // q_tile), -(-T // k_tile)
    out = np.zeros((max(nq, 1), max(nk, 1)), np.int8)
    _load().oracle_tile_kinds(_ptr(pln, _i32p), n, _ptr(f, _i32p), _ptr(b, _i32p), q_tile, k_tile,
                              _ptr(out, _i8p))
    return out[:nq, :nk]


def prefill_bwd(pages, q, k, v, dout, scale, q_rows=None, k_rows=None):
    """Gradients of the packed prefill for upstream gradient ``dout`` (Sec. 3.2 visibility,
    App. C.1 scatter-add of shared rows). Returns fp64 (dQ [nq][Hq][d], dK [nk][Hkv][d],
    dV [nk][Hkv][d]) for the packed query rows ``q_rows`` and key rows ``k_rows`` (default: all)."""
    pln, n, f, b = _flat(pages)
    q, k, v, g = _f32(q), _f32(k), _f32(v), _f32(dout)
    T, Hq, d = q.shape
    Hkv = k.shape[1]
    assert k.shape == (T, Hkv, d) and v.shape == (T, Hkv, d) and g.shape == q.shape and Hq % Hkv == 0
    qs = np.ascontiguousarray(np.arange(T) if q_rows is None else np.asarray(q_rows), np.int64)
    ks = np.ascontiguousarray(np.arange(T) if k_rows is None else np.asarray(k_rows), np.int64)
    assert ((qs >= 0) & (qs < T)).all() and ((ks >= 0) & (ks < T)).all()
    dq = np.zeros((len(qs), Hq, d), np.float64)
    dk = np.zeros((len(ks), Hkv, d), np.float64)
    dv = np.zeros((len(ks), Hkv, d), np.float64)
    guard = lambda a: a if a.size else np.zeros(1, a.dtype)
    if T:
        _load().oracle_prefill_bwd(_ptr(pln, _i32p), n, _ptr(f, _i32p), _ptr(b, _i32p), _ptr(q, _f32p),
                                   _ptr(k, _f32p), _ptr(v, _f32p), _ptr(g, _f32p), Hq, Hkv, d, float(scale),
                                   len(qs), _ptr(guard(qs), _i64p), len(ks), _ptr(guard(ks), _i64p),
                                   _ptr(guard(dq), _f64p), _ptr(guard(dk), _f64p), _ptr(guard(dv), _f64p))
    return dq, dk, dv


# --------------------------------------------------------------------------------------------
# FP8 (E4M3) KV cache: see padoc_oracle.c, "FP8 (E4M3) KV cache"
# --------------------------------------------------------------------------------------------

def e4m3_encode(x) -> np.ndarray:
    """E4M3 codes (uint8) of fp32 values: nearest, ties to even, saturating at 448, NaN -> 0x7F."""
    a = np.ascontiguousarray(np.asarray(x, np.float32))
    out = np.zeros(a.shape, np.uint8)
    _load().oracle_e4m3_encode(_ptr(a, _f32p), a.size, _ptr(out, _u8p))
    return out


def e4m3_decode(codes) -> np.ndarray:
    """fp64 values of E4M3 codes (NaN for 0x7F / 0xFF)."""
    c = np.ascontiguousarray(np.asarray(codes, np.uint8))
    out = np.zeros(c.shape, np.float64)
    _load().oracle_e4m3_decode(_ptr(c, _u8p), c.size, _ptr(out, _f64p))
    return out


def quantize_kv_blocks(pool):
    """pool fp32 [num_blocks][Hkv][block][d] -> (codes uint8 same shape, scales fp32 [num_blocks][Hkv]);
    scale = amax / 448 per (block, head), 0 for an all-zero one."""
    x = _f32(pool)
    nb, hkv, bs, d = x.shape
    codes = np.zeros(x.shape, np.uint8)
    scales = np.zeros((nb, hkv), np.float32)
    _load().oracle_quantize_kv_blocks(_ptr(x, _f32p), nb, hkv, bs, d, _ptr(codes, _u8p), _ptr(scales, _f32p))
    return codes, scales


def dequantize_kv_blocks(codes, scales) -> np.ndarray:
    """code_value * scale per (block, head), exact in fp64."""
    c = np.ascontiguousarray(np.asarray(codes, np.uint8))
    sc = np.ascontiguousarray(np.asarray(scales, np.float32))
    nb, hkv, bs, d = c.shape
    out = np.zeros(c.shape, np.float64)
    _load().oracle_dequantize_kv_blocks(_ptr(c, _u8p), _ptr(sc, _f32p), nb, hkv, bs, d, _ptr(out, _f64p))
    return out


def append_kv_quantized(codes, scales, slots, rows):
    """Appends rows [count][Hkv][d] (fp32 values) to slots (block * block + row) of a quantized pool,
    one at a time in order, with the scale rule of padoc_oracle.c:oracle_append_kv_quantized (the
    scale grows to amax / 448 of the rows so far; earlier rows are re-encoded when it grows; a
    block's row 0 starts it afresh). Returns new (codes, scales); the inputs are not changed."""
    c = np.ascontiguousarray(np.array(codes, np.uint8, copy=True))
    sc = np.ascontiguousarray(np.array(scales, np.float32, copy=True))
    nb, hkv, bs, d = c.shape
    sl = np.ascontiguousarray(np.asarray(slots, np.int32))
    x = _f32(rows)
    assert x.shape == (len(sl), hkv, d)
    if len(sl):
        _load().oracle_append_kv_quantized(_ptr(c, _u8p), _ptr(sc, _f32p), nb, hkv, bs, d, _ptr(sl, _i32p), len(sl),
                                           _ptr(x, _f32p))
    return c, sc


def decode_f64(stream_page, shared_len, priv_len, page_off, priv_off, stream_k, stream_v, priv_k, priv_v, q, scale):
    """``decode`` over fp64 K/V rows (e.g. a dequantized cache); q fp32-exact (bf16 or fp32)."""
    sp = np.ascontiguousarray(np.asarray(stream_page, np.int32))
    sh = np.ascontiguousarray(np.asarray(shared_len, np.int32))
    pl = np.ascontiguousarray(np.asarray(priv_len, np.int32))
    po = np.ascontiguousarray(np.asarray(page_off, np.int64))
    vo = np.ascontiguousarray(np.asarray(priv_off, np.int64))
    sk, sv, pk, pv = (np.ascontiguousarray(np.asarray(a, np.float64)) for a in (stream_k, stream_v, priv_k, priv_v))
    qq = _f32(q)
    S, Hq, d = qq.shape
    Hkv = sk.shape[1] if sk.size else pk.shape[1]
    guard = lambda a: a if a.size else np.zeros((1, Hkv, d), np.float64)
    sk, sv, pk, pv = guard(sk), guard(sv), guard(pk), guard(pv)
    o = np.zeros((S, Hq, d), np.float64)
    lse = np.zeros((S, Hq), np.float64)
    if S:
        _load().oracle_decode_f64(S, _ptr(sp, _i32p), _ptr(sh, _i32p), _ptr(pl, _i32p), _ptr(po, _i64p),
                                  _ptr(vo, _i64p), _ptr(sk, _f64p), _ptr(sv, _f64p), _ptr(pk, _f64p),
                                  _ptr(pv, _f64p), _ptr(qq, _f32p), Hq, Hkv, d, float(scale),
                                  _ptr(o, _f64p), _ptr(lse, _f64p))
    return o, lse


def decode_paged(pages, pool_k, pool_v, page_table, stream_table, q, scale, layout_streams: bool = False,
                 block_size: int = 16):
    """One decode step read through the paged layout: pool_k / pool_v [num_blocks][Hkv][block][d]
    (any real dtype; fp64 for a dequantized cache), page_table [pages][stride] (the block of each
    block_size rows of the page's shared stream), stream_table [streams][stride] (each stream's
    private rows from block offset 0). Streams and their cutoffs as ``decode_streams``; the rows each
    stream sees are gathered block by block and attended in fp64 with ``decode_f64``."""
    sp, sh, pl = decode_streams(pages, layout_streams)
    pk_ = np.asarray(pool_k, np.float64) if not hasattr(pool_k, "numpy") else pool_k.double().numpy()
    pv_ = np.asarray(pool_v, np.float64) if not hasattr(pool_v, "numpy") else pool_v.double().numpy()
    pt, st = np.asarray(page_table), np.asarray(stream_table)

    def rows(pool, table_row, n):
        out = [pool[int(table_row[t // block_size]), :, t % block_size, :] for t in range(n)]
        return np.stack(out) if out else np.zeros((0,) + pool.shape[1:2] + pool.shape[3:], np.float64)

    plen = [(pg[0] + pg[1]) if isinstance(pg, tuple) else pg.prefix_len + pg.layout_len for pg in pages]
    page_off = np.concatenate([[0], np.cumsum(plen)[:-1]]).astype(np.int64)
    priv_off = np.concatenate([[0], np.cumsum(pl.astype(np.int64))[:-1]]).astype(np.int64) if len(pl) else np.zeros(0, np.int64)
    sk = np.concatenate([rows(pk_, pt[p], plen[p]) for p in range(len(pages))]) if pages else np.zeros((0,))
    sv = np.concatenate([rows(pv_, pt[p], plen[p]) for p in range(len(pages))]) if pages else np.zeros((0,))
    prk = np.concatenate([rows(pk_, st[i], int(pl[i])) for i in range(len(pl))]) if len(pl) else np.zeros((0,))
    prv = np.concatenate([rows(pv_, st[i], int(pl[i])) for i in range(len(pl))]) if len(pl) else np.zeros((0,))
    return decode_f64(sp, sh, pl, page_off, priv_off, sk, sv, prk, prv, q, scale)
