"""One decode step and one packed prefill through the padoc_attn C ABI, for callers holding torch
tensors. Host work here is the C1 planners (in the library) and host<->device copies of their
integer outputs; every attention step runs in the library's CUDA kernels.
"""
from __future__ import annotations

from typing import List, Optional

import numpy as np
import torch

from . import padoc_attn as pa


class DecodePlan:
    """Decode plan (C1) uploaded to the device, with its split-K workspace (C4)."""

    def __init__(self, pages, num_q_heads: int, num_kv_heads: int, head_dim: int, device, block_size: int = 16,
                 layout_streams: bool = False, split_tokens: int = 0, tc_ctas: int = 0, warp_ctas: int = 0):
        self.cfg = pa.make_decode_config(num_q_heads, num_kv_heads, head_dim, block_size, layout_streams, split_tokens,
                                         tc_ctas, warp_ctas)
        plan, self.info = pa.padoc_build_decode_plan(pages, self.cfg)
        self.plan_host = plan
        self.plan_dev = torch.from_numpy(plan.copy()).to(device)
        ws = pa.padoc_decode_workspace_size(self.info)
        self.workspace = torch.empty(max(ws, 256), dtype=torch.uint8, device=device)

    @property
    def num_streams(self) -> int:
        return self.info.num_streams

    def run(self, k_pool, v_pool, page_table, stream_table, q, scale, out, lse, stream=None):
        pa.padoc_branch_decode_attn(k_pool, v_pool, self.info, self.plan_dev, page_table, stream_table, q, scale,
                                    out, lse, self.workspace, stream)


class PrefillPlan:
    """Spans and tile map (C1) of a packed prefill, uploaded to the device."""

    def __init__(self, pages, dtype: torch.dtype, head_dim: int, device):
        code = pa.PADOC_DTYPE_BF16 if dtype == torch.bfloat16 else pa.PADOC_DTYPE_F32
        self.q_tile, self.k_tile = pa.padoc_prefill_tile_shape(code, head_dim)
        self.spans_host = pa.padoc_build_query_spans(pages)
        self.row_ptr_host, self.k_tiles_host, self.kinds_host = pa.padoc_build_tile_map(pages, self.q_tile, self.k_tile)
        self.T = int(self.spans_host.shape[0])
        self.spans = torch.from_numpy(self.spans_host.copy()).to(device)
        self.row_ptr = torch.from_numpy(self.row_ptr_host.copy()).to(device)
        nnz = max(len(self.k_tiles_host), 1)
        self.k_tiles = torch.zeros(nnz, dtype=torch.int32, device=device)
        self.kinds = torch.zeros(nnz, dtype=torch.int8, device=device)
        if len(self.k_tiles_host):
            self.k_tiles.copy_(torch.from_numpy(self.k_tiles_host.copy()))
            self.kinds.copy_(torch.from_numpy(self.kinds_host.copy()))

    def run(self, q, k, v, scale, out, lse, stream=None):
        pa.padoc_ancestor_prefill_attn(q, k, v, self.spans, self.row_ptr, self.k_tiles, self.kinds, scale, out, lse,
                                       self.q_tile, self.k_tile, stream)


class PrefillBwdPlan:
    """Spans, the query-major and key-major tile maps (C1) and the workspace of a packed prefill's
    backward, on the device."""

    def __init__(self, pages, dtype: torch.dtype, head_dim: int, num_q_heads: int, device):
        code = pa.PADOC_DTYPE_BF16 if dtype == torch.bfloat16 else pa.PADOC_DTYPE_F32
        (qq, qk), (kq, kk) = pa.padoc_prefill_bwd_tile_shapes(code, head_dim)
        spans = pa.padoc_build_query_spans(pages)
        self.T = int(spans.shape[0])
        up = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a if len(a) else np.zeros(1, dt))).to(device)
        self.spans = torch.from_numpy(spans.copy()).to(device)
        row_ptr, k_tiles, kinds = pa.padoc_build_tile_map(pages, qq, qk)
        col_ptr, q_tiles, kkinds, order = pa.padoc_build_key_tile_map(pages, kq, kk)
        self._keep = [up(row_ptr, np.int32), up(k_tiles, np.int32), up(kinds, np.int8),
                      up(col_ptr, np.int32), up(q_tiles, np.int32), up(kkinds, np.int8), up(order, np.int32)]
        self.q_map = pa.make_tile_map_dev(*self._keep[:3], qq, qk)
        self.k_map = pa.make_tile_map_dev(*self._keep[3:6], kq, kk, order=self._keep[6])
        ws = pa.padoc_prefill_bwd_workspace_size(self.T, num_q_heads)
        self.workspace = torch.empty(max(ws, 256), dtype=torch.uint8, device=device)

    def run(self, q, k, v, out, dout, lse, scale, dq, dk, dv, stream=None):
        pa.padoc_ancestor_prefill_bwd(q, k, v, out, dout, lse, self.spans, self.q_map, self.k_map, scale, dq, dk, dv,
                                      self.workspace, stream)


def visible_pairs(pages) -> int:
    """Visible (query, key) pairs of a packed prefill, summed in closed form per page."""
    n = 0
    for pg in pages:
        P, L = pg.prefix_len, pg.layout_len
        M = P + L
        n += M * (M + 1) // 2
        for f, b in zip(pg.fork_offset, pg.branch_len):
            n += b * (P + f) + b * (b + 1) // 2
    return n


def shard_pages(num_pages: int, rank: int, world: int) -> List[int]:
    """Pages of one rank when pages are split across ranks (pages never see each other, so a
    rank's pages need nothing from any other rank): contiguous, sizes differing by at most one."""
    if world < 1 or not (0 <= rank < world):
        raise ValueError("bad rank/world")
    base, extra = divmod(num_pages, world)
    lo = rank * base + min(rank, extra)
    return list(range(lo, lo + base + (1 if rank < extra else 0)))
