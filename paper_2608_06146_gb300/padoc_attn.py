"""Python binding of the padoc_attn C ABI (include/padoc_attn.h): argument marshalling only.

Every function has the name of the C entry point it calls. Device buffers are torch CUDA tensors
(PyTorch supplies memory and streams); every step of the computation runs in the library's CUDA
kernels. There is no fallback: if the shared library is missing or a call fails, an exception is
raised.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "libpadoc_attn.so")

PADOC_OK = 0
PADOC_DTYPE_F32 = 0
PADOC_DTYPE_BF16 = 1
PADOC_TILE_PARTIAL = 1
PADOC_TILE_FULL = 2

_STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported combination", 3: "workspace too small",
           4: "CUDA error", 5: "device-side check failed", 6: "output capacity too small"}


class PadocError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} failed: {_STATUS.get(status, status)} (status {status})")


class padoc_page(ctypes.Structure):
    _fields_ = [("prefix_len", ctypes.c_int32), ("layout_len", ctypes.c_int32), ("num_branches", ctypes.c_int32),
                ("fork_offset", ctypes.POINTER(ctypes.c_int32)), ("branch_len", ctypes.POINTER(ctypes.c_int32))]


class padoc_kv_pool(ctypes.Structure):
    _fields_ = [("k_pool", ctypes.c_void_p), ("v_pool", ctypes.c_void_p), ("num_blocks", ctypes.c_int32),
                ("block_size", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("dtype", ctypes.c_int)]


class padoc_decode_config(ctypes.Structure):
    _fields_ = [("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("block_size", ctypes.c_int32), ("layout_streams", ctypes.c_int32), ("split_tokens", ctypes.c_int32),
                ("tc_ctas", ctypes.c_int32), ("warp_ctas", ctypes.c_int32)]


class padoc_kv_pool_e4m3(ctypes.Structure):
    _fields_ = [("k_codes", ctypes.c_void_p), ("v_codes", ctypes.c_void_p), ("k_scales", ctypes.c_void_p),
                ("v_scales", ctypes.c_void_p), ("num_blocks", ctypes.c_int32), ("block_size", ctypes.c_int32),
                ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32)]


class padoc_stream_desc(ctypes.Structure):
    _fields_ = [("page", ctypes.c_int32), ("shared_len", ctypes.c_int32), ("private_len", ctypes.c_int32)]


class padoc_prefill_chunk(ctypes.Structure):
    _fields_ = [("page", ctypes.c_int32), ("shared_len", ctypes.c_int32), ("private_start", ctypes.c_int32),
                ("num_tokens", ctypes.c_int32)]


class padoc_tile_map_dev(ctypes.Structure):
    _fields_ = [("ptr", ctypes.c_void_p), ("idx", ctypes.c_void_p), ("kind", ctypes.c_void_p),
                ("order", ctypes.c_void_p), ("q_tile", ctypes.c_int32), ("k_tile", ctypes.c_int32)]


class padoc_decode_plan(ctypes.Structure):
    _fields_ = [("cfg", padoc_decode_config), ("num_pages", ctypes.c_int32), ("num_streams", ctypes.c_int32),
                ("num_items", ctypes.c_int32), ("num_tc_items", ctypes.c_int32), ("tc_ctas", ctypes.c_int32),
                ("num_warps", ctypes.c_int32),
                ("num_slots", ctypes.c_int32),
                ("max_page_blocks", ctypes.c_int32), ("max_stream_blocks", ctypes.c_int32),
                ("max_stream_slots", ctypes.c_int32),
                ("plan_ints", ctypes.c_int64), ("off_stream_page", ctypes.c_int64), ("off_shared_len", ctypes.c_int64),
                ("off_private_len", ctypes.c_int64), ("off_slot_ptr", ctypes.c_int64), ("off_items", ctypes.c_int64),
                ("off_page_len", ctypes.c_int64), ("off_cta_ptr", ctypes.c_int64), ("off_warp_ptr", ctypes.c_int64),
                ("kv_tokens", ctypes.c_int64), ("off_merge_keys", ctypes.c_int64), ("num_merge_keys", ctypes.c_int32),
                ("reserved", ctypes.c_int32)]


class padoc_mpd_step(ctypes.Structure):
    _fields_ = [("num_streams", ctypes.c_int32), ("num_pages", ctypes.c_int32), ("page_stride", ctypes.c_int32),
                ("stream_stride", ctypes.c_int32), ("off_plan", ctypes.c_int64), ("off_page_table", ctypes.c_int64),
                ("off_stream_table", ctypes.c_int64), ("off_slots", ctypes.c_int64), ("off_rows", ctypes.c_int64), ("off_first_blocks", ctypes.c_int64),
                ("off_stream_ids", ctypes.c_int64), ("upload_words", ctypes.c_int64), ("total_words", ctypes.c_int64),
                ("plan", padoc_decode_plan)]


class padoc_mpd_run_args(ctypes.Structure):
    _fields_ = [("k_src", ctypes.c_void_p), ("v_src", ctypes.c_void_p), ("q_src", ctypes.c_void_p),
                ("src_total", ctypes.c_int64), ("src_row_of_stream", ctypes.c_void_p),
                ("num_stream_ids", ctypes.c_int32), ("scale", ctypes.c_float), ("out", ctypes.c_void_p),
                ("lse", ctypes.c_void_p), ("out_rows", ctypes.c_int32), ("ids_capacity", ctypes.c_int32),
                ("stream_ids", ctypes.c_void_p), ("stream", ctypes.c_void_p)]


_lib = None
_i32p = ctypes.POINTER(ctypes.c_int32)
_i64p = ctypes.POINTER(ctypes.c_int64)
_i8p = ctypes.POINTER(ctypes.c_int8)
_vp = ctypes.c_void_p


def load_library(path: Optional[str] = None):
    """Load libpadoc_attn.so (built in-tree by paper_2608_06146_gb300.build). Raises if absent."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or LIB_PATH
    if not os.path.exists(path):
        raise RuntimeError(f"padoc_attn CUDA library not built: {path} is missing (run __graft_entry__.build())")
    lib = ctypes.CDLL(path)
    P = ctypes.POINTER(padoc_page)
    sig = {
        "padoc_packed_size": [P, ctypes.c_int32, _i64p],
        "padoc_build_query_spans": [P, ctypes.c_int32, _i32p, ctypes.c_int64],
        "padoc_prefill_tile_shape": [ctypes.c_int, ctypes.c_int32, _i32p, _i32p],
        "padoc_tile_map_size": [P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, _i64p, _i64p],
        "padoc_build_tile_map": [P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, _i32p, _i32p, _i8p, ctypes.c_int64],
        "padoc_decode_plan_size": [P, ctypes.c_int32, ctypes.POINTER(padoc_decode_config), _i64p],
        "padoc_build_decode_plan": [P, ctypes.c_int32, ctypes.POINTER(padoc_decode_config), _i32p, ctypes.c_int64,
                                    ctypes.POINTER(padoc_decode_plan)],
        "padoc_decode_workspace_size": [ctypes.POINTER(padoc_decode_plan), ctypes.POINTER(ctypes.c_size_t)],
        "padoc_branch_decode_attn": [ctypes.POINTER(padoc_kv_pool), ctypes.POINTER(padoc_decode_plan), _vp, _vp,
                                     ctypes.c_int32, _vp, ctypes.c_int32, _vp, ctypes.c_float, _vp, _vp, _vp,
                                     ctypes.c_size_t, _vp],
        "padoc_branch_decode_attn_noalloc": [ctypes.POINTER(padoc_kv_pool), ctypes.POINTER(padoc_decode_plan), _vp,
                                             _vp, ctypes.c_int32, _vp, ctypes.c_int32, _vp, ctypes.c_float, _vp, _vp,
                                             _vp],
        "padoc_splitk_combine": [_vp, _vp, ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, ctypes.c_int, _vp, _vp, _vp],
        "padoc_ancestor_prefill_attn": [_vp, _vp, _vp, ctypes.c_int, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                        ctypes.c_int32, _vp, _vp, _vp, _vp, ctypes.c_int32, ctypes.c_int32,
                                        ctypes.c_float, _vp, _vp, _vp],
        "padoc_build_key_tile_map": [P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, _i32p, _i32p, _i8p, _i32p,
                                     ctypes.c_int64],
        "padoc_prefill_bwd_tile_shapes": [ctypes.c_int, ctypes.c_int32, _i32p, _i32p, _i32p, _i32p],
        "padoc_prefill_bwd_workspace_size": [ctypes.c_int64, ctypes.c_int32, ctypes.POINTER(ctypes.c_size_t)],
        "padoc_ancestor_prefill_bwd": [_vp, _vp, _vp, _vp, _vp, _vp, ctypes.c_int, ctypes.c_int64, ctypes.c_int32,
                                       ctypes.c_int32, ctypes.c_int32, _vp, ctypes.POINTER(padoc_tile_map_dev),
                                       ctypes.POINTER(padoc_tile_map_dev), ctypes.c_float, _vp, _vp, _vp, _vp,
                                       ctypes.c_size_t, _vp],
        "padoc_decode_plan_size_streams": [_i32p, ctypes.c_int32, ctypes.POINTER(padoc_stream_desc), ctypes.c_int32,
                                           ctypes.POINTER(padoc_decode_config), _i64p],
        "padoc_build_decode_plan_streams": [_i32p, ctypes.c_int32, ctypes.POINTER(padoc_stream_desc), ctypes.c_int32,
                                            ctypes.POINTER(padoc_decode_config), _i32p, ctypes.c_int64,
                                            ctypes.POINTER(padoc_decode_plan)],
        "padoc_chunk_prefill_plan_size": [_i32p, ctypes.c_int32, ctypes.POINTER(padoc_prefill_chunk), ctypes.c_int32,
                                          ctypes.POINTER(padoc_decode_config), _i64p],
        "padoc_build_chunk_prefill_plan": [_i32p, ctypes.c_int32, ctypes.POINTER(padoc_prefill_chunk), ctypes.c_int32,
                                           ctypes.POINTER(padoc_decode_config), _i32p, ctypes.c_int64,
                                           ctypes.POINTER(padoc_decode_plan)],
        "padoc_expand_chunk_table": [ctypes.POINTER(padoc_prefill_chunk), ctypes.c_int32, _i32p, ctypes.c_int32, _i32p,
                                     ctypes.c_int32, ctypes.c_int64],
        "padoc_mpd_create": [ctypes.c_int32, ctypes.c_int32, _i32p, ctypes.POINTER(_vp)],
        "padoc_mpd_destroy": [_vp],
        "padoc_mpd_add_page": [_vp, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, _i32p, _i32p, _i32p],
        "padoc_mpd_begin_step": [_vp, _i32p, _i32p, _i32p, ctypes.c_int32],
        "padoc_mpd_step_shape": [_vp, _i32p, _i32p, _i32p, _i32p],
        "padoc_mpd_step_tables": [_vp, _i32p, ctypes.POINTER(padoc_stream_desc), _i32p, ctypes.c_int32, _i32p,
                                  ctypes.c_int32],
        "padoc_mpd_end_step": [_vp, _vp, _vp, ctypes.c_int32, _vp, ctypes.c_int32, _i32p],
        "padoc_mpd_status": [_vp, _i32p, _i32p, _i32p],
        "padoc_mpd_prepare_step": [_vp, ctypes.POINTER(padoc_decode_config), _i32p, ctypes.c_int64,
                                   ctypes.POINTER(padoc_mpd_step)],
        "padoc_append_inputs": [ctypes.POINTER(padoc_kv_pool), _vp, _vp, _vp, ctypes.c_int64, ctypes.c_int32, _vp, _vp,
                                _vp, ctypes.c_int32, _vp],
        "padoc_mpd_launch_step": [ctypes.POINTER(padoc_mpd_step), _vp, _vp, ctypes.c_int64,
                                  ctypes.POINTER(padoc_kv_pool), _vp, _vp, _vp, ctypes.c_int64, _vp, ctypes.c_float, _vp,
                                  _vp, _vp, ctypes.c_size_t, _vp],
        "padoc_mpd_runner_create": [_vp, ctypes.POINTER(padoc_decode_config), ctypes.POINTER(padoc_kv_pool),
                                    ctypes.POINTER(_vp)],
        "padoc_mpd_runner_destroy": [_vp],
        "padoc_mpd_runner_step": [_vp, ctypes.POINTER(padoc_mpd_run_args), _i32p, _i64p],
        "padoc_mpd_runner_last_step": [_vp, ctypes.POINTER(padoc_mpd_step), ctypes.POINTER(_i32p)],
        "padoc_selftest_tcgen05": [_vp, _vp, _vp, _vp, _vp, _vp, _vp],
        "padoc_selftest_wait_timeout": [ctypes.c_int32, ctypes.c_int32, _vp, _vp],
        "padoc_advance_decode_plan": [_i32p, ctypes.POINTER(padoc_decode_plan), _i32p, ctypes.c_int32],
        "padoc_launch_decode_step": [ctypes.POINTER(padoc_kv_pool), ctypes.POINTER(padoc_decode_plan), _vp,
                                     ctypes.c_int64, ctypes.c_int64, ctypes.c_int32, ctypes.c_int64, ctypes.c_int32,
                                     _vp, ctypes.c_int64, _vp, _vp, ctypes.c_float, _vp, _vp, _vp, _vp, _vp,
                                     ctypes.c_size_t, _vp, _vp, _vp, _vp, _vp, _vp],
        "padoc_quantize_kv_blocks": [ctypes.POINTER(padoc_kv_pool_e4m3), _vp, _vp, _vp, ctypes.c_int32, _vp],
        "padoc_append_inputs_e4m3": [ctypes.POINTER(padoc_kv_pool_e4m3), _vp, _vp, _vp, ctypes.c_int64, ctypes.c_int32,
                                     _vp, _vp, _vp, ctypes.c_int32, _vp],
        "padoc_branch_decode_attn_e4m3": [ctypes.POINTER(padoc_kv_pool_e4m3), ctypes.POINTER(padoc_decode_plan), _vp,
                                          _vp, ctypes.c_int32, _vp, ctypes.c_int32, _vp, ctypes.c_float, _vp, _vp,
                                          _vp, ctypes.c_size_t, _vp],
        "padoc_check_device_errors": [_vp],
        "padoc_last_device_error": [_i32p, _i32p],
        "padoc_status_string": [ctypes.c_int],
        "padoc_version": [],
    }
    for name, args in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = ctypes.c_int
    lib.padoc_status_string.restype = ctypes.c_char_p
    lib.padoc_last_device_error.restype = None
    lib.padoc_mpd_destroy.restype = None
    lib.padoc_mpd_runner_destroy.restype = None
    _lib = lib
    return lib


def exported_symbols() -> Sequence[str]:
    return [n for n in ("padoc_packed_size", "padoc_build_query_spans", "padoc_prefill_tile_shape",
                        "padoc_tile_map_size", "padoc_build_tile_map", "padoc_decode_plan_size",
                        "padoc_build_decode_plan", "padoc_decode_workspace_size", "padoc_branch_decode_attn",
                        "padoc_branch_decode_attn_noalloc",
                        "padoc_splitk_combine", "padoc_ancestor_prefill_attn", "padoc_build_key_tile_map",
                        "padoc_prefill_bwd_tile_shapes", "padoc_prefill_bwd_workspace_size",
                        "padoc_ancestor_prefill_bwd", "padoc_decode_plan_size_streams",
                        "padoc_build_decode_plan_streams", "padoc_chunk_prefill_plan_size",
                        "padoc_build_chunk_prefill_plan", "padoc_expand_chunk_table",
                        "padoc_mpd_create", "padoc_mpd_destroy",
                        "padoc_mpd_add_page", "padoc_mpd_begin_step", "padoc_mpd_step_shape",
                        "padoc_mpd_step_tables", "padoc_mpd_end_step", "padoc_mpd_status", "padoc_mpd_prepare_step",
                        "padoc_mpd_launch_step", "padoc_mpd_runner_create", "padoc_mpd_runner_destroy",
                        "padoc_mpd_runner_step", "padoc_mpd_runner_last_step",
                        "padoc_append_inputs",
                        "padoc_selftest_tcgen05", "padoc_selftest_wait_timeout",
                        "padoc_quantize_kv_blocks", "padoc_append_inputs_e4m3", "padoc_branch_decode_attn_e4m3",
                        "padoc_advance_decode_plan", "padoc_launch_decode_step",
                        "padoc_check_device_errors",
                        "padoc_last_device_error", "padoc_status_string", "padoc_version")]


def _check(fn: str, st: int):
    if st != PADOC_OK:
        raise PadocError(fn, st)


_PAGE_DTYPE = np.dtype({"names": ["prefix_len", "layout_len", "num_branches", "fork_offset", "branch_len"],
                        "formats": [np.int32, np.int32, np.int32, np.uint64, np.uint64],
                        "offsets": [0, 4, 8, 16, 24], "itemsize": ctypes.sizeof(padoc_page)})


class _Pages:
    """C array of padoc_page built with vectorized numpy (one pass over the pages); keeps the
    concatenated fork-offset and branch-length arrays alive.

    Public as PageArray: a caller that plans every step (a decode loop whose branches grow by one
    token per step) keeps one and updates its arrays in place (``lens``: every page's branch lengths
    back to back; ``forks``: their fork offsets; ``rec["prefix_len"]`` / ``rec["layout_len"]``) instead
    of marshalling Python page objects again; the page and branch counts are fixed."""

    def __init__(self, pages):
        import itertools
        n = len(pages)
        counts = np.fromiter((len(pg.branch_len) for pg in pages), np.int64, count=n)
        total = int(counts.sum())
        self.forks = np.fromiter(itertools.chain.from_iterable(pg.fork_offset for pg in pages), np.int32, count=total)
        self.lens = np.fromiter(itertools.chain.from_iterable(pg.branch_len for pg in pages), np.int32, count=total)
        if total == 0:
            self.forks = np.zeros(1, np.int32)
            self.lens = np.zeros(1, np.int32)
        offs = np.zeros(max(n, 1), np.int64)
        if n > 1:
            offs[1:] = np.cumsum(counts)[:-1]
        rec = np.zeros(max(n, 1), _PAGE_DTYPE)
        rec["prefix_len"][:n] = np.fromiter((pg.prefix_len for pg in pages), np.int32, count=n)
        rec["layout_len"][:n] = np.fromiter((pg.layout_len for pg in pages), np.int32, count=n)
        rec["num_branches"][:n] = counts
        rec["fork_offset"][:n] = self.forks.ctypes.data + 4 * offs[:n]
        rec["branch_len"][:n] = self.lens.ctypes.data + 4 * offs[:n]
        self.rec = rec
        self.arr = ctypes.cast(rec.ctypes.data, ctypes.POINTER(padoc_page))
        self.n = n


PageArray = _Pages


def _as_pages(pages) -> _Pages:
    return pages if isinstance(pages, _Pages) else _Pages(pages)


_raw_stream = None


def _stream_ptr(stream):
    """The cudaStream_t of ``stream`` (a torch stream or a raw handle); None: torch's current stream."""
    global _raw_stream
    if stream is None:
        import torch
        if _raw_stream is None:
            get, dev = getattr(torch._C, "_cuda_getCurrentRawStream", None), getattr(torch._C, "_cuda_getDevice", None)
            _raw_stream = (lambda: get(dev())) if get and dev else (lambda: torch.cuda.current_stream().cuda_stream)
        return _raw_stream()
    return getattr(stream, "cuda_stream", stream)


def _dtype_code(t):
    import torch
    if t.dtype == torch.bfloat16:
        return PADOC_DTYPE_BF16
    if t.dtype == torch.float32:
        return PADOC_DTYPE_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def _dev(t, name):
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous CUDA tensor")
    return t.data_ptr()


# ------------------------------------------------------------------------------------------------
# C1: descriptors
# ------------------------------------------------------------------------------------------------

def padoc_packed_size(pages) -> int:
    lib, P = load_library(), _as_pages(pages)
    t = ctypes.c_int64()
    _check("padoc_packed_size", lib.padoc_packed_size(P.arr, P.n, ctypes.byref(t)))
    return t.value


def padoc_build_query_spans(pages) -> np.ndarray:
    lib, P = load_library(), _as_pages(pages)
    T = padoc_packed_size(pages)
    out = np.zeros((max(T, 1), 4), np.int32)
    _check("padoc_build_query_spans", lib.padoc_build_query_spans(P.arr, P.n, out.ctypes.data_as(_i32p), T))
    return out[:T]


def padoc_prefill_tile_shape(dtype: int, head_dim: int):
    lib = load_library()
    a, b = ctypes.c_int32(), ctypes.c_int32()
    _check("padoc_prefill_tile_shape", lib.padoc_prefill_tile_shape(dtype, head_dim, ctypes.byref(a), ctypes.byref(b)))
    return a.value, b.value


def padoc_tile_map_size(pages, q_tile: int, k_tile: int):
    lib, P = load_library(), _as_pages(pages)
    a, b = ctypes.c_int64(), ctypes.c_int64()
    _check("padoc_tile_map_size", lib.padoc_tile_map_size(P.arr, P.n, q_tile, k_tile, ctypes.byref(a), ctypes.byref(b)))
    return a.value, b.value


def padoc_build_tile_map(pages, q_tile: int, k_tile: int):
    """Returns (row_ptr int32 [q_tiles+1], k_tiles int32 [nnz], kinds int8 [nnz])."""
    lib, P = load_library(), _as_pages(pages)
    nqt, nnz = padoc_tile_map_size(pages, q_tile, k_tile)
    row_ptr = np.zeros(nqt + 1, np.int32)
    kt = np.zeros(max(nnz, 1), np.int32)
    kind = np.zeros(max(nnz, 1), np.int8)
    _check("padoc_build_tile_map", lib.padoc_build_tile_map(P.arr, P.n, q_tile, k_tile, row_ptr.ctypes.data_as(_i32p),
                                                            kt.ctypes.data_as(_i32p), kind.ctypes.data_as(_i8p), nnz))
    return row_ptr, kt[:nnz], kind[:nnz]


def padoc_build_key_tile_map(pages, q_tile: int, k_tile: int):
    """Returns (col_ptr int32 [k_tiles+1], q_tiles int32 [nnz], kinds int8 [nnz], k_order int32 [k_tiles])."""
    lib, P = load_library(), _as_pages(pages)
    T = padoc_packed_size(pages)
    _, nnz = padoc_tile_map_size(pages, q_tile, k_tile)
    nkt = -(-T // k_tile)
    col_ptr = np.zeros(nkt + 1, np.int32)
    qt = np.zeros(max(nnz, 1), np.int32)
    kind = np.zeros(max(nnz, 1), np.int8)
    order = np.zeros(max(nkt, 1), np.int32)
    _check("padoc_build_key_tile_map",
           lib.padoc_build_key_tile_map(P.arr, P.n, q_tile, k_tile, col_ptr.ctypes.data_as(_i32p),
                                        qt.ctypes.data_as(_i32p), kind.ctypes.data_as(_i8p),
                                        order.ctypes.data_as(_i32p), nnz))
    return col_ptr, qt[:nnz], kind[:nnz], order[:nkt]


def padoc_prefill_bwd_tile_shapes(dtype: int, head_dim: int):
    """Returns ((dq_q_tile, dq_k_tile), (dkv_q_tile, dkv_k_tile))."""
    lib = load_library()
    a, b, c, d = (ctypes.c_int32() for _ in range(4))
    _check("padoc_prefill_bwd_tile_shapes",
           lib.padoc_prefill_bwd_tile_shapes(dtype, head_dim, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c),
                                             ctypes.byref(d)))
    return (a.value, b.value), (c.value, d.value)


# ------------------------------------------------------------------------------------------------
# Decode
# ------------------------------------------------------------------------------------------------

def make_decode_config(num_q_heads, num_kv_heads, head_dim, block_size=16, layout_streams=False, split_tokens=0,
                       tc_ctas=0, warp_ctas=0):
    return padoc_decode_config(num_q_heads, num_kv_heads, head_dim, block_size, int(bool(layout_streams)), split_tokens,
                               tc_ctas, warp_ctas)


def padoc_decode_plan_size(pages, cfg: padoc_decode_config) -> int:
    lib, P = load_library(), _as_pages(pages)
    n = ctypes.c_int64()
    _check("padoc_decode_plan_size", lib.padoc_decode_plan_size(P.arr, P.n, ctypes.byref(cfg), ctypes.byref(n)))
    return n.value


def padoc_build_decode_plan(pages, cfg: padoc_decode_config, out=None):
    """Returns (plan blob int32 numpy array, padoc_decode_plan host summary). ``out`` may be an int32
    numpy array (e.g. a view of pinned host memory) that receives the blob; a view of it is returned."""
    lib, P = load_library(), _as_pages(pages)
    info = padoc_decode_plan()
    if out is not None:   # one planner pass when the caller's buffer is large enough
        st = lib.padoc_build_decode_plan(P.arr, P.n, ctypes.byref(cfg), out.ctypes.data_as(_i32p), out.size,
                                         ctypes.byref(info))
        if st == PADOC_OK:
            return out[:info.plan_ints], info
        if st != 6:   # PADOC_ERR_CAPACITY
            _check("padoc_build_decode_plan", st)
    n = ctypes.c_int64()
    _check("padoc_decode_plan_size", lib.padoc_decode_plan_size(P.arr, P.n, ctypes.byref(cfg), ctypes.byref(n)))
    n = n.value
    out = np.zeros(max(n, 1), np.int32)
    _check("padoc_build_decode_plan", lib.padoc_build_decode_plan(P.arr, P.n, ctypes.byref(cfg),
                                                                  out.ctypes.data_as(_i32p), n, ctypes.byref(info)))
    return out[:n], info


_STREAM_DTYPE = np.dtype([("page", np.int32), ("shared_len", np.int32), ("private_len", np.int32)])


def _stream_arr(streams):
    """streams: numpy array of _STREAM_DTYPE (or an int32 [S][3] array)."""
    a = np.ascontiguousarray(streams)
    if a.dtype != _STREAM_DTYPE:
        a = np.ascontiguousarray(np.asarray(a, np.int32).reshape(-1, 3)).view(_STREAM_DTYPE).reshape(-1)
    return a, ctypes.cast(a.ctypes.data, ctypes.POINTER(padoc_stream_desc))


def padoc_decode_plan_size_streams(page_len, streams, cfg: padoc_decode_config) -> int:
    lib = load_library()
    pl = np.ascontiguousarray(page_len, np.int32)
    sa, sp = _stream_arr(streams)
    n = ctypes.c_int64()
    _check("padoc_decode_plan_size_streams",
           lib.padoc_decode_plan_size_streams(pl.ctypes.data_as(_i32p), pl.size, sp, sa.size, ctypes.byref(cfg),
                                              ctypes.byref(n)))
    return n.value


def padoc_build_decode_plan_streams(page_len, streams, cfg: padoc_decode_config, out=None):
    """The decode plan of an explicit stream list (page_len int32 [pages]; streams [S] of
    (page, shared_len, private_len)). Returns (plan blob, padoc_decode_plan); ``out`` as in
    padoc_build_decode_plan."""
    lib = load_library()
    pl = np.ascontiguousarray(page_len, np.int32)
    sa, sp = _stream_arr(streams)
    info = padoc_decode_plan()
    if out is not None:
        st = lib.padoc_build_decode_plan_streams(pl.ctypes.data_as(_i32p), pl.size, sp, sa.size, ctypes.byref(cfg),
                                                 out.ctypes.data_as(_i32p), out.size, ctypes.byref(info))
        if st == PADOC_OK:
            return out[:info.plan_ints], info
        if st != 6:
            _check("padoc_build_decode_plan_streams", st)
    n = padoc_decode_plan_size_streams(pl, sa, cfg)
    out = np.zeros(max(n, 1), np.int32)
    _check("padoc_build_decode_plan_streams",
           lib.padoc_build_decode_plan_streams(pl.ctypes.data_as(_i32p), pl.size, sp, sa.size, ctypes.byref(cfg),
                                               out.ctypes.data_as(_i32p), n, ctypes.byref(info)))
    return out[:n], info


_CHUNK_DTYPE = np.dtype([("page", np.int32), ("shared_len", np.int32), ("private_start", np.int32),
                         ("num_tokens", np.int32)])


def _chunk_arr(chunks):
    a = np.ascontiguousarray(np.asarray(chunks, np.int32).reshape(-1, 4)).view(_CHUNK_DTYPE).reshape(-1)
    return a, ctypes.cast(a.ctypes.data, ctypes.POINTER(padoc_prefill_chunk))


def padoc_build_chunk_prefill_plan(page_len, chunks, cfg: padoc_decode_config):
    """Plan of a chunked prefill: page_len int32 [pages]; chunks [C] of (page, shared_len, private_start,
    num_tokens). Returns (plan blob, padoc_decode_plan)."""
    lib = load_library()
    pl = np.ascontiguousarray(page_len, np.int32)
    ca, cp = _chunk_arr(chunks)
    n = ctypes.c_int64()
    _check("padoc_chunk_prefill_plan_size",
           lib.padoc_chunk_prefill_plan_size(pl.ctypes.data_as(_i32p), pl.size, cp, ca.size, ctypes.byref(cfg),
                                             ctypes.byref(n)))
    out = np.zeros(max(n.value, 1), np.int32)
    info = padoc_decode_plan()
    _check("padoc_build_chunk_prefill_plan",
           lib.padoc_build_chunk_prefill_plan(pl.ctypes.data_as(_i32p), pl.size, cp, ca.size, ctypes.byref(cfg),
                                              out.ctypes.data_as(_i32p), n.value, ctypes.byref(info)))
    return out[:n.value], info


def padoc_expand_chunk_table(chunks, chunk_table, stream_stride=None):
    """Per-token stream block table [tokens][stride] from one row per chunk ([chunks][chunk_stride])."""
    lib = load_library()
    ca, cp = _chunk_arr(chunks)
    ct = np.ascontiguousarray(chunk_table, np.int32)
    stride = ct.shape[1] if stream_stride is None else stream_stride
    rows = int(ca["num_tokens"].sum())
    out = np.zeros((max(rows, 1), stride), np.int32)
    _check("padoc_expand_chunk_table",
           lib.padoc_expand_chunk_table(cp, ca.size, ct.ctypes.data_as(_i32p), ct.shape[1], out.ctypes.data_as(_i32p),
                                        stride, rows))
    return out[:rows]


def padoc_decode_workspace_size(info: padoc_decode_plan) -> int:
    lib = load_library()
    b = ctypes.c_size_t()
    _check("padoc_decode_workspace_size", lib.padoc_decode_workspace_size(ctypes.byref(info), ctypes.byref(b)))
    return b.value


def padoc_branch_decode_attn(k_pool, v_pool, info: padoc_decode_plan, plan_dev, page_table, stream_table, q, scale,
                             out, lse, workspace=None, stream=None):
    """k_pool/v_pool: [num_blocks][Hkv][16][d]; page_table [pages][stride]; stream_table [streams][stride]
    (int32 CUDA tensors); q/out: [streams][Hq][d]; lse: fp32 [streams][Hq]; workspace: uint8 CUDA tensor."""
    lib = load_library()
    pool = padoc_kv_pool(_dev(k_pool, "k_pool"), _dev(v_pool, "v_pool"), k_pool.shape[0], k_pool.shape[2],
                         k_pool.shape[1], k_pool.shape[3], _dtype_code(k_pool))
    ws = _dev(workspace, "workspace") if workspace is not None else None
    wsb = workspace.numel() * workspace.element_size() if workspace is not None else 0
    st = lib.padoc_branch_decode_attn(ctypes.byref(pool), ctypes.byref(info), _dev(plan_dev, "plan_dev"),
                                      _dev(page_table, "page_table"), page_table.shape[1],
                                      _dev(stream_table, "stream_table"), stream_table.shape[1], _dev(q, "q"),
                                      float(scale), _dev(out, "out"), _dev(lse, "lse"), ws, wsb, _stream_ptr(stream))
    _check("padoc_branch_decode_attn", st)


def padoc_advance_decode_plan(plan, info: padoc_decode_plan, private_len) -> bool:
    """Patches ``plan`` (int32 numpy host blob) and ``info`` in place for new private lengths of the
    same streams; False (nothing changed) when a new plan is needed."""
    lib = load_library()
    pl = np.ascontiguousarray(np.asarray(private_len, np.int32))
    st = lib.padoc_advance_decode_plan(plan.ctypes.data_as(_i32p), ctypes.byref(info), pl.ctypes.data_as(_i32p),
                                       pl.size)
    if st == 6:
        return False
    _check("padoc_advance_decode_plan", st)
    return True


def padoc_launch_decode_step(k_pool, v_pool, info: padoc_decode_plan, stage, stage_words: int, off_page_table: int,
                             page_stride: int, off_stream_table: int, stream_stride: int, dev_ints, q_host, q_dev,
                             scale, out_dev, lse_dev, out_host, lse_host, workspace, stream=None, copy_in=None,
                             copy_out=None, ev_free=None, ev_in=None, ev_dec=None):
    """One decode step from host inputs: stage (pinned int32 CPU tensor: plan blob, page table, stream
    table), q_host (pinned) -> device, decode, out / lse -> out_host / lse_host (pinned); no sync.
    With copy_in / copy_out (torch streams) and the buffer set's three torch events, the copies run
    on those streams, ordered by the events (see the C header)."""
    ev = lambda e: None if e is None else e.cuda_event
    lib = load_library()
    pool = padoc_kv_pool(_dev(k_pool, "k_pool"), _dev(v_pool, "v_pool"), k_pool.shape[0], k_pool.shape[2],
                         k_pool.shape[1], k_pool.shape[3], _dtype_code(k_pool))
    st = lib.padoc_launch_decode_step(ctypes.byref(pool), ctypes.byref(info), stage.data_ptr(), int(stage_words),
                                      int(off_page_table), int(page_stride), int(off_stream_table), int(stream_stride),
                                      _dev(dev_ints, "dev_ints"), dev_ints.numel(), q_host.data_ptr(),
                                      _dev(q_dev, "q_dev"), float(scale), _dev(out_dev, "out_dev"),
                                      _dev(lse_dev, "lse_dev"), out_host.data_ptr(), lse_host.data_ptr(),
                                      _dev(workspace, "workspace"), workspace.numel() * workspace.element_size(),
                                      _stream_ptr(stream), None if copy_in is None else _stream_ptr(copy_in),
                                      None if copy_out is None else _stream_ptr(copy_out), ev(ev_free), ev(ev_in),
                                      ev(ev_dec))
    _check("padoc_launch_decode_step", st)


class DecodeStep:
    """One buffer set of a decode loop's host side with its arguments marshalled once: each call
    patches the set's host plan for the streams' new private lengths (padoc_advance_decode_plan;
    False, with nothing launched, when a new plan is needed) and runs padoc_launch_decode_step. The
    arguments are those of the two functions; the tensors, arrays and streams must stay alive and
    unmoved while the object is used."""

    def __init__(self, k_pool, v_pool, info: padoc_decode_plan, stage, stage_words: int, plan_ints: int,
                 off_page_table: int, page_stride: int, off_stream_table: int, stream_stride: int, dev_ints, q_host,
                 q_dev, scale, out_dev, lse_dev, out_host, lse_host, workspace, private_len, stream=None,
                 copy_in=None, copy_out=None, ev_free=None, ev_in=None, ev_dec=None):
        lib = load_library()
        self._f_adv, self._f_launch = lib.padoc_advance_decode_plan, lib.padoc_launch_decode_step
        self._pool = padoc_kv_pool(_dev(k_pool, "k_pool"), _dev(v_pool, "v_pool"), k_pool.shape[0], k_pool.shape[2],
                                   k_pool.shape[1], k_pool.shape[3], _dtype_code(k_pool))
        self._info = info
        plan = stage.numpy()[:plan_ints]
        self._pl = np.ascontiguousarray(np.asarray(private_len, np.int32))
        self._keep = (k_pool, v_pool, stage, dev_ints, q_host, q_dev, out_dev, lse_dev, out_host, lse_host, workspace,
                      plan, stream, copy_in, copy_out, ev_free, ev_in, ev_dec)
        ev = lambda e: None if e is None else e.cuda_event
        self._adv_args = (plan.ctypes.data_as(_i32p), ctypes.byref(info), self._pl.ctypes.data_as(_i32p), self._pl.size)
        self._launch_args = (ctypes.byref(self._pool), ctypes.byref(info), stage.data_ptr(), int(stage_words),
                             int(off_page_table), int(page_stride), int(off_stream_table), int(stream_stride),
                             _dev(dev_ints, "dev_ints"), dev_ints.numel(), q_host.data_ptr(), _dev(q_dev, "q_dev"),
                             float(scale), _dev(out_dev, "out_dev"), _dev(lse_dev, "lse_dev"), out_host.data_ptr(),
                             lse_host.data_ptr(), _dev(workspace, "workspace"),
                             workspace.numel() * workspace.element_size(), _stream_ptr(stream),
                             None if copy_in is None else _stream_ptr(copy_in),
                             None if copy_out is None else _stream_ptr(copy_out), ev(ev_free), ev(ev_in), ev(ev_dec))

    def __call__(self) -> bool:
        st = self._f_adv(*self._adv_args)
        if st == 6:
            return False
        _check("padoc_advance_decode_plan", st)
        _check("padoc_launch_decode_step", self._f_launch(*self._launch_args))
        return True


PADOC_STATIC_WORKSPACE_BYTES = 32 << 20


def padoc_branch_decode_attn_noalloc(k_pool, v_pool, info: padoc_decode_plan, plan_dev, page_table, stream_table, q,
                                     scale, out, lse, stream=None):
    """padoc_branch_decode_attn for callers that cannot allocate device memory: the split-K partials
    go to the library's fixed 32 MiB device array (shared by every call; serialize calls)."""
    lib = load_library()
    pool = padoc_kv_pool(_dev(k_pool, "k_pool"), _dev(v_pool, "v_pool"), k_pool.shape[0], k_pool.shape[2],
                         k_pool.shape[1], k_pool.shape[3], _dtype_code(k_pool))
    st = lib.padoc_branch_decode_attn_noalloc(ctypes.byref(pool), ctypes.byref(info), _dev(plan_dev, "plan_dev"),
                                              _dev(page_table, "page_table"), page_table.shape[1],
                                              _dev(stream_table, "stream_table"), stream_table.shape[1], _dev(q, "q"),
                                              float(scale), _dev(out, "out"), _dev(lse, "lse"), _stream_ptr(stream))
    _check("padoc_branch_decode_attn_noalloc", st)


def padoc_splitk_combine(part_o, part_lse, out, lse=None, stream=None):
    """part_o fp32 [S][rows][d], part_lse fp32 [S][rows] -> out [rows][d] (bf16 or fp32), lse fp32 [rows]."""
    lib = load_library()
    S, R, d = part_o.shape
    st = lib.padoc_splitk_combine(_dev(part_o, "part_o"), _dev(part_lse, "part_lse"), S, R, d, _dtype_code(out),
                                  _dev(out, "out"), _dev(lse, "lse"), _stream_ptr(stream))
    _check("padoc_splitk_combine", st)


# ------------------------------------------------------------------------------------------------
# Algorithm 1: the masked parallel decoding loop
# ------------------------------------------------------------------------------------------------

class Mpd:
    """The loop's host-side scheduler (padoc_mpd_*). Methods return numpy int32 arrays."""

    def __init__(self, num_blocks: int, block_size: int = 16, block_order=None):
        self._lib = load_library()
        h = _vp()
        order = None if block_order is None else np.ascontiguousarray(block_order, np.int32)
        _check("padoc_mpd_create", self._lib.padoc_mpd_create(num_blocks, block_size,
                                                              None if order is None else order.ctypes.data_as(_i32p),
                                                              ctypes.byref(h)))
        self._h = h
        self.block_size = block_size
        self._cap = 0
        self._ids = self._slots = None
        self._ev_cap = 64
        self._nf = np.zeros(self._ev_cap, np.int32)
        self._eos = np.zeros(self._ev_cap, np.uint8)
        self._nf_p, self._eos_p = self._nf.ctypes.data, self._eos.ctypes.data
        self._new = np.zeros(256, np.int32)
        self._new_p = self._new.ctypes.data
        self._k = ctypes.c_int32()
        self._k_ref = ctypes.byref(self._k)

    def close(self):
        if self._h:
            self._lib.padoc_mpd_destroy(self._h)
            self._h = _vp()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def add_page(self, prefix_len: int, num_forks: int = 0, layout_eos: bool = False):
        """Returns (page id, prefix slots int32 [P], new stream ids int32 [1 + num_forks]; the first
        is the layout stream's, -1 with layout_eos)."""
        pid = ctypes.c_int32()
        slots = np.zeros(max(prefix_len, 1), np.int32)
        new = np.zeros(1 + num_forks, np.int32)
        _check("padoc_mpd_add_page", self._lib.padoc_mpd_add_page(self._h, prefix_len, num_forks, int(bool(layout_eos)),
                                                                  ctypes.byref(pid), slots.ctypes.data_as(_i32p),
                                                                  new.ctypes.data_as(_i32p)))
        return pid.value, slots[:prefix_len], new

    def begin_step(self):
        """Returns (stream ids, append slots) of the step, both int32 [C]."""
        lp, ls, fb = self.status()
        if ls > self._cap:
            self._cap = max(ls, 2 * self._cap, 64)
            self._ids = np.zeros(self._cap, np.int32)
            self._slots = np.zeros(self._cap, np.int32)
        c = ctypes.c_int32()
        ids = self._ids if self._ids is not None else np.zeros(1, np.int32)
        slots = self._slots if self._slots is not None else np.zeros(1, np.int32)
        _check("padoc_mpd_begin_step", self._lib.padoc_mpd_begin_step(self._h, ctypes.byref(c), ids.ctypes.data_as(_i32p),
                                                                      slots.ctypes.data_as(_i32p), max(self._cap, 0)))
        return ids[:c.value].copy(), slots[:c.value].copy()

    def step_shape(self):
        a, b, c, d = (ctypes.c_int32() for _ in range(4))
        _check("padoc_mpd_step_shape", self._lib.padoc_mpd_step_shape(self._h, ctypes.byref(a), ctypes.byref(b),
                                                                      ctypes.byref(c), ctypes.byref(d)))
        return a.value, b.value, c.value, d.value

    def step_tables(self, page_stride=None, stream_stride=None):
        """Returns (page_len int32 [pages], streams [S] of _STREAM_DTYPE, page_table int32 [pages][stride],
        stream_table int32 [S][stride])."""
        npg, ns, mp, ms = self.step_shape()
        page_stride = max(mp, 1) if page_stride is None else page_stride
        stream_stride = max(ms, 1) if stream_stride is None else stream_stride
        page_len = np.zeros(max(npg, 1), np.int32)
        streams = np.zeros(max(ns, 1), _STREAM_DTYPE)
        pt = np.zeros((max(npg, 1), page_stride), np.int32)
        stt = np.zeros((max(ns, 1), stream_stride), np.int32)
        _check("padoc_mpd_step_tables",
               self._lib.padoc_mpd_step_tables(self._h, page_len.ctypes.data_as(_i32p),
                                               ctypes.cast(streams.ctypes.data, ctypes.POINTER(padoc_stream_desc)),
                                               pt.ctypes.data_as(_i32p), page_stride, stt.ctypes.data_as(_i32p),
                                               stream_stride))
        return page_len[:npg], streams[:ns], pt[:npg], stt[:ns]

    def end_step(self, num_forks=None, eos=None, num_streams=None):
        """num_forks int32 [C], eos bool/uint8 [C] (None = all zero). Returns the new branches' ids.
        The events are copied into arrays kept here, whose addresses are marshalled once."""
        n = num_streams
        if n is None:
            n = len(num_forks) if num_forks is not None else len(eos) if eos is not None else 0
        if n > self._ev_cap:
            self._ev_cap = max(n, 2 * self._ev_cap, 64)
            self._nf = np.zeros(self._ev_cap, np.int32)
            self._eos = np.zeros(self._ev_cap, np.uint8)
            self._nf_p, self._eos_p = self._nf.ctypes.data, self._eos.ctypes.data
        fp = ep = None
        if num_forks is not None:
            self._nf[:n] = num_forks
            fp = self._nf_p
        if eos is not None:
            self._eos[:n] = eos
            ep = self._eos_p
        while True:
            st = self._lib.padoc_mpd_end_step(self._h, fp, ep, n, self._new_p, self._new.size, self._k_ref)
            if st != 6 or fp is None:
                break
            self._new = np.zeros(max(2 * self._new.size, int(self._nf[:n].sum())), np.int32)   # nothing changed
            self._new_p = self._new.ctypes.data
        _check("padoc_mpd_end_step", st)
        return self._new[:self._k.value].copy()

    def prepare_step(self, cfg: padoc_decode_config, stage: np.ndarray) -> padoc_mpd_step:
        """padoc_mpd_prepare_step into ``stage`` (int32 numpy array, e.g. a view of pinned memory).
        Raises PadocError (status 6) when the stage is too small; step.total_words is then set on
        the error's ``step`` attribute."""
        st = padoc_mpd_step()
        code = self._lib.padoc_mpd_prepare_step(self._h, ctypes.byref(cfg), stage.ctypes.data_as(_i32p), stage.size,
                                                ctypes.byref(st))
        if code != PADOC_OK:
            err = PadocError("padoc_mpd_prepare_step", code)
            err.step = st
            raise err
        return st

    def status(self):
        """(live pages, live streams, free blocks)."""
        a, b, c = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
        _check("padoc_mpd_status", self._lib.padoc_mpd_status(self._h, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)))
        return a.value, b.value, c.value


def padoc_mpd_launch_step(step: padoc_mpd_step, stage, dev_ints, pool: padoc_kv_pool, k_src, v_src, q_src, q_dst,
                          scale, out, lse, workspace, stream=None):
    """stage: pinned int32 CPU tensor holding the prepared step (None: dev_ints already holds it);
    dev_ints: int32 CUDA tensor; pool: a padoc_kv_pool (make_kv_pool); other tensors as in
    padoc_append_inputs / padoc_branch_decode_attn."""
    lib = load_library()
    st = lib.padoc_mpd_launch_step(ctypes.byref(step), None if stage is None else stage.data_ptr(),
                                   _dev(dev_ints, "dev_ints"), dev_ints.numel(),
                                   ctypes.byref(pool), _dev(k_src, "k_src"), _dev(v_src, "v_src"), _dev(q_src, "q_src"),
                                   k_src.shape[0], _dev(q_dst, "q_dst"), float(scale), _dev(out, "out"),
                                   _dev(lse, "lse"), _dev(workspace, "workspace"),
                                   workspace.numel() * workspace.element_size(), _stream_ptr(stream))
    _check("padoc_mpd_launch_step", st)


class MpdRunner:
    """padoc_mpd_runner_*: the loop's per-step host work in one library call. The runner owns its
    staging and device buffers; the scheduler and the pool (their padoc_kv_pool and tensors) must
    outlive it. ``step`` takes the source rows as an int32 table indexed by stream id."""

    def __init__(self, mpd: Mpd, cfg: padoc_decode_config, pool: padoc_kv_pool):
        self._lib = load_library()
        self._mpd, self._cfg, self._pool = mpd, cfg, pool   # kept alive
        h = _vp()
        _check("padoc_mpd_runner_create", self._lib.padoc_mpd_runner_create(mpd._h, ctypes.byref(cfg),
                                                                            ctypes.byref(pool), ctypes.byref(h)))
        self._h = h
        self._args = padoc_mpd_run_args()
        self._args_ref = ctypes.byref(self._args)
        self._n = ctypes.c_int32()
        self._n_ref = ctypes.byref(self._n)
        self._up = ctypes.c_int64()
        self._up_ref = ctypes.byref(self._up)
        self._ids = np.zeros(64, np.int32)
        self._args.ids_capacity, self._args.stream_ids = self._ids.size, self._ids.ctypes.data
        self._src = None
        self._outs = {}

    def close(self):
        if self._h:
            self._lib.padoc_mpd_runner_destroy(self._h)
            self._h = _vp()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def step(self, k_src, v_src, q_src, row_of_stream: np.ndarray, scale: float, out, lse, stream=None):
        """One step: returns (C, stream ids int32 [C], a view of the runner's array valid until the
        next step). out [rows >= C][Hq][d] and lse fp32 [rows][Hq] receive the outputs in step order;
        row_of_stream: int32 [ids] (host), the source row of each live stream's input. Arrays are
        checked the first time they are seen (the runner keeps the last few)."""
        a = self._args
        src = self._src
        if src is None or src[0] is not k_src or src[1] is not v_src or src[2] is not q_src or \
                src[3] is not row_of_stream:
            self._set_sources(k_src, v_src, q_src, row_of_stream)
        o = self._outs.get((id(out), id(lse)))
        if o is None or o[0] is not out or o[1] is not lse:
            o = self._set_outputs(out, lse)
        a.out, a.lse, a.out_rows = o[2], o[3], o[4]
        a.scale = scale
        a.stream = _stream_ptr(stream)
        _check("padoc_mpd_runner_step", self._lib.padoc_mpd_runner_step(self._h, self._args_ref, self._n_ref,
                                                                        self._up_ref))
        n = self._n.value
        return n, self._ids[:n]

    @property
    def upload_bytes(self) -> int:
        """Bytes the last step copied to the device."""
        return self._up.value

    def _set_sources(self, k_src, v_src, q_src, row_of_stream):
        c = self._cfg
        dt = PADOC_DTYPE_BF16 if self._pool.dtype == PADOC_DTYPE_BF16 else PADOC_DTYPE_F32
        for t, nm in ((k_src, "k_src"), (v_src, "v_src"), (q_src, "q_src")):
            _dev(t, nm)
            if _dtype_code(t) != dt:
                raise TypeError(f"{nm} must have the pool's dtype")
        if (tuple(k_src.shape[1:]) != (c.num_kv_heads, c.head_dim) or tuple(v_src.shape) != tuple(k_src.shape) or
                tuple(q_src.shape[1:]) != (c.num_q_heads, c.head_dim) or q_src.shape[0] != k_src.shape[0]):
            raise ValueError("k_src/v_src [rows][Hkv][d], q_src [rows][Hq][d]")
        if not isinstance(row_of_stream, np.ndarray) or row_of_stream.dtype != np.int32 or \
                not row_of_stream.flags.c_contiguous:
            raise ValueError("row_of_stream must be a contiguous int32 numpy array")
        a = self._args
        a.k_src, a.v_src, a.q_src = k_src.data_ptr(), v_src.data_ptr(), q_src.data_ptr()
        a.src_total = k_src.shape[0]
        a.src_row_of_stream = row_of_stream.ctypes.data
        a.num_stream_ids = row_of_stream.size
        self._src = (k_src, v_src, q_src, row_of_stream)

    def _set_outputs(self, out, lse):
        c = self._cfg
        dt = PADOC_DTYPE_BF16 if self._pool.dtype == PADOC_DTYPE_BF16 else PADOC_DTYPE_F32
        _dev(out, "out")
        _dev(lse, "lse")
        if _dtype_code(out) != dt:
            raise TypeError("out must have the pool's dtype")
        if str(lse.dtype) != "torch.float32":
            raise TypeError("lse must be float32")
        if tuple(out.shape[1:]) != (c.num_q_heads, c.head_dim) or lse.dim() != 2 or lse.shape[1] != c.num_q_heads:
            raise ValueError("out [rows][Hq][d], lse [rows][Hq]")
        cap = min(int(out.shape[0]), int(lse.shape[0]))
        if self._ids.size < cap:
            self._ids = np.zeros(cap, np.int32)
            self._args.ids_capacity, self._args.stream_ids = self._ids.size, self._ids.ctypes.data
        if len(self._outs) >= 8:
            self._outs.clear()
        o = (out, lse, out.data_ptr(), lse.data_ptr(), cap)
        self._outs[(id(out), id(lse))] = o
        return o

    def last_step(self):
        """(padoc_mpd_step, its staging buffer as an int32 numpy array [total_words])."""
        st = padoc_mpd_step()
        p = _i32p()
        _check("padoc_mpd_runner_last_step", self._lib.padoc_mpd_runner_last_step(self._h, ctypes.byref(st),
                                                                                  ctypes.byref(p)))
        return st, np.ctypeslib.as_array(p, (max(int(st.total_words), 1),))


def make_kv_pool(k_pool, v_pool) -> padoc_kv_pool:
    """padoc_kv_pool over pool tensors [num_blocks][Hkv][16][d] (the caller keeps them alive)."""
    return padoc_kv_pool(_dev(k_pool, "k_pool"), _dev(v_pool, "v_pool"), k_pool.shape[0], k_pool.shape[2],
                         k_pool.shape[1], k_pool.shape[3], _dtype_code(k_pool))


class E4M3Pool:
    """An FP8 (E4M3) paged KV pool on the device: codes uint8 [num_blocks][Hkv][16][d] for K and V and
    fp32 scales [num_blocks][Hkv] (torch tensors owned here), and its padoc_kv_pool_e4m3."""

    def __init__(self, num_blocks: int, num_kv_heads: int, head_dim: int, device, block_size: int = 16):
        import torch
        shape = (num_blocks, num_kv_heads, block_size, head_dim)
        self.k_codes = torch.zeros(shape, dtype=torch.uint8, device=device)
        self.v_codes = torch.zeros(shape, dtype=torch.uint8, device=device)
        self.k_scales = torch.zeros((num_blocks, num_kv_heads), dtype=torch.float32, device=device)
        self.v_scales = torch.zeros((num_blocks, num_kv_heads), dtype=torch.float32, device=device)
        self.c = padoc_kv_pool_e4m3(_dev(self.k_codes, "k_codes"), _dev(self.v_codes, "v_codes"),
                                    _dev(self.k_scales, "k_scales"), _dev(self.v_scales, "v_scales"), num_blocks,
                                    block_size, num_kv_heads, head_dim)

    @property
    def num_blocks(self) -> int:
        return self.c.num_blocks


def padoc_quantize_kv_blocks(pool: E4M3Pool, k_src, v_src, dst_blocks, stream=None):
    """Whole bf16 blocks k_src / v_src [count][Hkv][16][d] into pool blocks dst_blocks (int32 CUDA tensor)."""
    lib = load_library()
    _check("padoc_quantize_kv_blocks", lib.padoc_quantize_kv_blocks(ctypes.byref(pool.c), _dev(k_src, "k_src"),
                                                                    _dev(v_src, "v_src"), _dev(dst_blocks, "dst_blocks"),
                                                                    dst_blocks.shape[0], _stream_ptr(stream)))


def padoc_append_inputs_e4m3(pool: E4M3Pool, k_src, v_src, slots, q_src=None, q_dst=None, src_rows=None, count=None,
                             stream=None):
    """padoc_append_inputs into an E4M3 pool (bf16 sources); the slots of one call in distinct blocks."""
    lib = load_library()
    n = slots.shape[0] if count is None else count
    hq = q_src.shape[1] if q_src is not None else 0
    st = lib.padoc_append_inputs_e4m3(ctypes.byref(pool.c), _dev(k_src, "k_src"), _dev(v_src, "v_src"),
                                      _dev(q_src, "q_src"), k_src.shape[0], hq, _dev(q_dst, "q_dst"),
                                      _dev(src_rows, "src_rows"), _dev(slots, "slots"), n, _stream_ptr(stream))
    _check("padoc_append_inputs_e4m3", st)


def padoc_branch_decode_attn_e4m3(pool: E4M3Pool, info: padoc_decode_plan, plan_dev, page_table, stream_table, q,
                                  scale, out, lse, workspace, stream=None):
    """padoc_branch_decode_attn over an E4M3 pool (q / out bf16 [streams][Hq][128], lse fp32)."""
    lib = load_library()
    st = lib.padoc_branch_decode_attn_e4m3(ctypes.byref(pool.c), ctypes.byref(info), _dev(plan_dev, "plan_dev"),
                                           _dev(page_table, "page_table"), page_table.shape[1],
                                           _dev(stream_table, "stream_table"), stream_table.shape[1], _dev(q, "q"),
                                           float(scale), _dev(out, "out"), _dev(lse, "lse"),
                                           _dev(workspace, "workspace"), workspace.numel() * workspace.element_size(),
                                           _stream_ptr(stream))
    _check("padoc_branch_decode_attn_e4m3", st)


def padoc_append_inputs(k_pool, v_pool, k_src, v_src, slots, q_src=None, q_dst=None, src_rows=None, count=None,
                        stream=None):
    """K/V rows (src_rows or 0..count-1) of k_src/v_src [rows][Hkv][d] into pool slots (int32 CUDA tensor);
    with q_src [rows][Hq][d], the same rows' queries into q_dst [count][Hq][d]."""
    lib = load_library()
    pool = padoc_kv_pool(_dev(k_pool, "k_pool"), _dev(v_pool, "v_pool"), k_pool.shape[0], k_pool.shape[2],
                         k_pool.shape[1], k_pool.shape[3], _dtype_code(k_pool))
    n = slots.shape[0] if count is None else count
    hq = q_src.shape[1] if q_src is not None else 0
    st = lib.padoc_append_inputs(ctypes.byref(pool), _dev(k_src, "k_src"), _dev(v_src, "v_src"), _dev(q_src, "q_src"),
                                 k_src.shape[0], hq, _dev(q_dst, "q_dst"), _dev(src_rows, "src_rows"),
                                 _dev(slots, "slots"), n, _stream_ptr(stream))
    _check("padoc_append_inputs", st)


# ------------------------------------------------------------------------------------------------
# Prefill
# ------------------------------------------------------------------------------------------------

def padoc_ancestor_prefill_attn(q, k, v, spans_dev, row_ptr_dev, k_tiles_dev, kinds_dev, scale, out, lse,
                                q_tile=128, k_tile=128, stream=None):
    """q/out [T][Hq][d]; k/v [T][Hkv][d]; spans_dev int32 [T][4]; tile map on the device (or None for fp32)."""
    lib = load_library()
    T, Hq, d = q.shape
    Hkv = k.shape[1]
    st = lib.padoc_ancestor_prefill_attn(_dev(q, "q"), _dev(k, "k"), _dev(v, "v"), _dtype_code(q), T, Hq, Hkv, d,
                                         _dev(spans_dev, "spans"), _dev(row_ptr_dev, "row_ptr"),
                                         _dev(k_tiles_dev, "k_tiles"), _dev(kinds_dev, "kinds"), q_tile, k_tile,
                                         float(scale), _dev(out, "out"), _dev(lse, "lse"), _stream_ptr(stream))
    _check("padoc_ancestor_prefill_attn", st)


def make_tile_map_dev(ptr, idx, kind, q_tile: int, k_tile: int, order=None) -> padoc_tile_map_dev:
    """A padoc_tile_map_dev over device tensors (the caller keeps them alive)."""
    return padoc_tile_map_dev(_dev(ptr, "ptr"), _dev(idx, "idx"), _dev(kind, "kind"),
                              _dev(order, "order") if order is not None else None, q_tile, k_tile)


def padoc_prefill_bwd_workspace_size(total_tokens: int, num_q_heads: int) -> int:
    lib = load_library()
    n = ctypes.c_size_t()
    _check("padoc_prefill_bwd_workspace_size",
           lib.padoc_prefill_bwd_workspace_size(total_tokens, num_q_heads, ctypes.byref(n)))
    return n.value


def padoc_ancestor_prefill_bwd(q, k, v, out, dout, lse, spans_dev, q_map: padoc_tile_map_dev,
                               k_map: padoc_tile_map_dev, scale, dq, dk, dv, workspace, stream=None):
    """Gradients of the packed prefill: q/out/dout/dq [T][Hq][d]; k/v/dk/dv [T][Hkv][d]; lse fp32 [T][Hq];
    workspace a uint8 device tensor of padoc_prefill_bwd_workspace_size bytes."""
    lib = load_library()
    T, Hq, d = q.shape
    Hkv = k.shape[1]
    st = lib.padoc_ancestor_prefill_bwd(_dev(q, "q"), _dev(k, "k"), _dev(v, "v"), _dev(out, "out"),
                                        _dev(dout, "dout"), _dev(lse, "lse"), _dtype_code(q), T, Hq, Hkv, d,
                                        _dev(spans_dev, "spans"), ctypes.byref(q_map), ctypes.byref(k_map),
                                        float(scale), _dev(dq, "dq"), _dev(dk, "dk"), _dev(dv, "dv"),
                                        _dev(workspace, "workspace"), workspace.numel() * workspace.element_size(),
                                        _stream_ptr(stream))
    _check("padoc_ancestor_prefill_bwd", st)


def padoc_selftest_tcgen05(a, bk, v, c1, c2, c3, stream=None):
    """c1 = a . bk^T, c2 = a . v and c3 = a . v (a from tensor memory) on the tensor cores
    (bf16 [128][128] inputs, fp32 outputs)."""
    lib = load_library()
    _check("padoc_selftest_tcgen05", lib.padoc_selftest_tcgen05(_dev(a, "a"), _dev(bk, "bk"), _dev(v, "v"),
                                                                _dev(c1, "c1"), _dev(c2, "c2"), _dev(c3, "c3"),
                                                                _stream_ptr(stream)))


def padoc_selftest_wait_timeout(limit_us: int, site: int, gave_up, stream=None):
    """One CTA's bounded wait on an mbarrier nothing arrives at, with a limit of limit_us; the
    device error word then holds code 2 with ``site``; gave_up (int32 CUDA tensor, zeroed by the
    caller) counts the threads whose wait gave up."""
    lib = load_library()
    _check("padoc_selftest_wait_timeout", lib.padoc_selftest_wait_timeout(int(limit_us), int(site),
                                                                          _dev(gave_up, "gave_up"),
                                                                          _stream_ptr(stream)))


def padoc_check_device_errors(stream=None):
    """Synchronizes the stream and raises PadocError if a kernel recorded a failed device check."""
    lib = load_library()
    st = lib.padoc_check_device_errors(_stream_ptr(stream))
    if st != PADOC_OK:
        code, detail = ctypes.c_int32(), ctypes.c_int32()
        lib.padoc_last_device_error(ctypes.byref(code), ctypes.byref(detail))
        err = PadocError("padoc_check_device_errors", st)
        err.device_code, err.device_detail = code.value, detail.value
        raise err


def padoc_status_string(status: int) -> str:
    return load_library().padoc_status_string(status).decode()


def padoc_version() -> int:
    return load_library().padoc_version()
