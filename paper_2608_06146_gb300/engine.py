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


class ChunkPrefillPlan:
    """Plan (C1) of a chunked prefill over the paged cache, uploaded: chunks of consecutive query
    tokens per stream (padoc_prefill_chunk rows), run by the decode kernels with the chunks' tokens
    as streams; ``chunk_table`` holds each chunk's private block ids (one row per chunk)."""

    def __init__(self, page_len, chunks, chunk_table, num_q_heads: int, num_kv_heads: int, head_dim: int, device,
                 block_size: int = 16, tc_ctas: int = 0, warp_ctas: int = 0):
        self.cfg = pa.make_decode_config(num_q_heads, num_kv_heads, head_dim, block_size, False, 0, tc_ctas, warp_ctas)
        self.chunks = np.ascontiguousarray(np.asarray(chunks, np.int32).reshape(-1, 4))
        plan, self.info = pa.padoc_build_chunk_prefill_plan(page_len, self.chunks, self.cfg)
        self.plan_dev = torch.from_numpy(plan.copy()).to(device)
        table = pa.padoc_expand_chunk_table(self.chunks, chunk_table,
                                            max(int(self.info.max_stream_blocks), np.asarray(chunk_table).shape[1], 1))
        self.stream_table = torch.from_numpy(table.copy()).to(device)
        ws = pa.padoc_decode_workspace_size(self.info)
        self.workspace = torch.empty(max(ws, 256), dtype=torch.uint8, device=device)

    @property
    def num_tokens(self) -> int:
        return self.info.num_streams

    def run(self, k_pool, v_pool, page_table, q, scale, out, lse, stream=None):
        """q / out: [tokens][Hq][d] in the chunks' token order; lse fp32 [tokens][Hq]."""
        pa.padoc_branch_decode_attn(k_pool, v_pool, self.info, self.plan_dev, page_table, self.stream_table, q, scale,
                                    out, lse, self.workspace, stream)


class MaskedParallelLoop:
    """Algorithm 1 (App. E.1) over the library: the host scheduler (padoc_mpd_*), the append kernel
    and the decode step on one paged KV pool, with device memory from torch.

    Per step the host asks the scheduler for the live streams and their input slots, builds the
    step's decode plan from the stream list, and sends slots, source rows, block tables and plan to
    the device in one copy from pinned memory (two staging buffers, so the host fills one while
    the previous step's copy may still read the other). The device then appends every input's K/V
    into the pool, lays out the queries and decodes every stream, all on one CUDA stream."""

    def __init__(self, num_blocks: int, num_q_heads: int, num_kv_heads: int, head_dim: int, dtype: torch.dtype,
                 device, block_order=None, block_size: int = 16, tc_ctas: int = 0, warp_ctas: int = 0,
                 split_tokens: int = 0):
        self.mpd = pa.Mpd(num_blocks, block_size, block_order)
        self.k_pool = torch.zeros((num_blocks, num_kv_heads, block_size, head_dim), dtype=dtype, device=device)
        self.v_pool = torch.zeros_like(self.k_pool)
        self._pool = pa.make_kv_pool(self.k_pool, self.v_pool)
        self.cfg = pa.make_decode_config(num_q_heads, num_kv_heads, head_dim, block_size, False, split_tokens,
                                         tc_ctas, warp_ctas)
        self.device, self.dtype = device, dtype
        self.num_q_heads, self.head_dim = num_q_heads, head_dim
        self._stage = [None, None]
        self._stage_free = [torch.cuda.Event(), torch.cuda.Event()]
        self._turn = 0
        self._ints = torch.empty(1024, dtype=torch.int32, device=device)
        self.workspace = torch.empty(256, dtype=torch.uint8, device=device)
        self.q_step = torch.empty((64, num_q_heads, head_dim), dtype=dtype, device=device)
        self.last_info = None
        self.last_step = None
        self.last_stage = None
        self.h2d_bytes = 0
        self._runner = None

    def _upload(self, parts, stream):
        """Copies int32 host arrays to the device in one transfer, each starting on a 128-byte
        boundary; returns device views."""
        offs, n = [], 0
        for a in parts:
            offs.append(n)
            n += (int(a.size) + 31) // 32 * 32
        b = self._turn & 1
        self._turn += 1
        self._stage_free[b].synchronize()
        if self._stage[b] is None or self._stage[b].numel() < n:
            self._stage[b] = torch.empty(max(n, 2 * (0 if self._stage[b] is None else self._stage[b].numel()), 4096),
                                         dtype=torch.int32).pin_memory()
        host = self._stage[b].numpy()
        for a, o in zip(parts, offs):
            host[o:o + a.size] = a.reshape(-1)
        if self._ints.numel() < n:
            self._ints = torch.empty(max(n, 2 * self._ints.numel()), dtype=torch.int32, device=self.device)
        with torch.cuda.stream(stream):
            self._ints[:n].copy_(self._stage[b][:n], non_blocking=True)
        self._stage_free[b].record(stream)
        self.h2d_bytes = 4 * n
        return [self._ints[o:o + a.size] for a, o in zip(parts, offs)]

    def add_page(self, prefix_len: int, num_forks: int, layout_eos: bool, k_src, v_src, src_rows, stream=None):
        """Admits a page: its prefix K/V (rows src_rows of k_src / v_src, device tensors [rows][Hkv][d])
        go into the blocks the scheduler gives it. Returns (page id, new stream ids)."""
        stream = stream or torch.cuda.current_stream()
        pid, slots, new = self.mpd.add_page(prefix_len, num_forks, layout_eos)
        if prefix_len > 0:
            slots_d, rows_d = self._upload([slots, np.asarray(src_rows, np.int32)], stream)
            pa.padoc_append_inputs(self.k_pool, self.v_pool, k_src, v_src, slots_d, src_rows=rows_d, count=prefix_len,
                                   stream=stream)
        return pid, new

    def step(self, k_src, v_src, q_src, rows_of, scale: float, out=None, lse=None, stream=None):
        """One iteration: every live stream appends its next input (rows_of(stream ids) gives the rows
        of k_src / v_src / q_src that hold them) and is decoded. Returns (stream ids, out [C][Hq][d],
        lse fp32 [C][Hq]); the caller ends the step with end_step. The host work is two library calls:
        padoc_mpd_prepare_step into a pinned staging buffer, and padoc_mpd_launch_step, which copies it
        to the device and launches the append and the decode."""
        stream = stream or torch.cuda.current_stream()
        b = self._turn & 1
        self._turn += 1
        self._stage_free[b].synchronize()
        if self._stage[b] is None:
            self._stage[b] = torch.empty(1 << 16, dtype=torch.int32).pin_memory()
        while True:
            try:
                st = self.mpd.prepare_step(self.cfg, self._stage[b].numpy())
                break
            except pa.PadocError as e:
                need = getattr(e, "step", None)
                if e.status != 6 or need is None or need.total_words <= self._stage[b].numel():
                    raise
                self._stage[b] = torch.empty(2 * int(need.total_words), dtype=torch.int32).pin_memory()
        host = self._stage[b].numpy()
        C = int(st.num_streams)
        ids = host[st.off_stream_ids:st.off_stream_ids + C].copy()
        host[st.off_rows:st.off_rows + C] = rows_of(ids)
        n = int(st.upload_words)
        if self._ints.numel() < n:
            self._ints = torch.empty(max(n, 2 * self._ints.numel()), dtype=torch.int32, device=self.device)
        self.h2d_bytes = 4 * n
        info = st.plan
        self.last_info = info
        self.last_step = st
        self.last_stage = host
        if C == 0:
            self._stage_free[b].record(stream)
            empty = torch.empty((0, self.num_q_heads), dtype=torch.float32, device=self.device)
            return ids, torch.empty((0, self.num_q_heads, self.head_dim), dtype=self.dtype, device=self.device), empty
        if self.q_step.shape[0] < C:
            self.q_step = torch.empty((max(C, 2 * self.q_step.shape[0]), self.num_q_heads, self.head_dim),
                                      dtype=self.dtype, device=self.device)
        ws = pa.padoc_decode_workspace_size(info)
        if self.workspace.numel() < ws:
            self.workspace = torch.empty(max(ws, 2 * self.workspace.numel()), dtype=torch.uint8, device=self.device)
        if out is None:
            out = torch.empty((C, self.num_q_heads, self.head_dim), dtype=self.dtype, device=self.device)
        if lse is None:
            lse = torch.empty((C, self.num_q_heads), dtype=torch.float32, device=self.device)
        # one library call: the stage's copy to the device, the append and the decode
        pa.padoc_mpd_launch_step(st, self._stage[b], self._ints, self._pool, k_src, v_src, q_src, self.q_step, scale,
                                 out, lse, self.workspace, stream)
        self._stage_free[b].record(stream)
        return ids, out, lse

    def run_step(self, k_src, v_src, q_src, row_of_stream, scale: float, out, lse, stream=None):
        """step() as one library call (padoc_mpd_runner_step): row_of_stream is an int32 numpy table
        of each live stream's source row indexed by stream id; out [rows][Hq][d] and lse [rows][Hq]
        (rows at least the live streams) receive the outputs in step order. Returns (C, stream ids
        int32 [C], valid until the next step); end the step with end_step."""
        if self._runner is None:
            self._runner = pa.MpdRunner(self.mpd, self.cfg, self._pool)
        n, ids = self._runner.step(k_src, v_src, q_src, row_of_stream, scale, out, lse, stream)
        self.h2d_bytes = self._runner.upload_bytes
        return n, ids

    def last_run_step(self):
        """(padoc_mpd_step, its staging words) of the last run_step."""
        return self._runner.last_step()

    def end_step(self, num_forks=None, eos=None, num_streams=None):
        """Each stream's output event (forks, EOS) in step order; returns the new branches' ids."""
        return self.mpd.end_step(num_forks, eos, num_streams)

    def status(self):
        return self.mpd.status()


def shard_pages(num_pages: int, rank: int, world: int) -> List[int]:
    """Pages of one rank when pages are split across ranks (pages never see each other, so a
    rank's pages need nothing from any other rank): contiguous, sizes differing by at most one."""
    if world < 1 or not (0 <= rank < world):
        raise ValueError("bad rank/world")
    base, extra = divmod(num_pages, world)
    lo = rank * base + min(rank, extra)
    return list(range(lo, lo + base + (1 if rank < extra else 0)))
