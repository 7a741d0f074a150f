"""The device entry points validate their arguments on the host before any launch: malformed calls
return INVALID_ARGUMENT (1), UNSUPPORTED (2) or WORKSPACE_TOO_SMALL (3) and touch no memory. These
calls use stand-in addresses that are never dereferenced because every case here is rejected
before the library reaches the device; the module skips itself where a GPU is visible, so that no
call with stand-in addresses can ever reach a launch."""
import ctypes

import pytest
import torch

from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import padoc_attn as pa

pytestmark = pytest.mark.skipif(torch.cuda.is_available(), reason="stand-in addresses are for machines without a GPU")

A = 1 << 20          # a 256-byte-aligned stand-in address
MIS = A + 4          # misaligned


@pytest.fixture(scope="module")
def lib():
    pbuild.build()
    return pa.load_library()


def _pool(block_size=16, hkv=2, d=128, dtype=pa.PADOC_DTYPE_BF16, k=A, v=A):
    return pa.padoc_kv_pool(k, v, 64, block_size, hkv, d, dtype)


def _decode_info(lib):
    from paper_2608_06146_gb300.inputs import PageSpec
    cfg = pa.make_decode_config(16, 2, 128)
    _, info = pa.padoc_build_decode_plan([PageSpec(40, 8, [3, 8], [5, 20])], cfg)
    return info


def test_decode_rejects_malformed_calls(lib):
    info = _decode_info(lib)
    call = lambda pool, plan=A, pt=A, pts=8, st=A, sts=8, q=A, scale=0.1, out=A, lse=A: lib.padoc_branch_decode_attn(
        ctypes.byref(pool) if pool is not None else None, ctypes.byref(info), plan, pt, pts, st, sts, q, scale, out,
        lse, A, 1 << 20, None)
    assert call(None) == 1                                  # no pool
    assert call(_pool(), plan=None) == 1                    # no plan
    assert call(_pool(block_size=32)) == 1                  # pool and plan disagree
    assert call(_pool(hkv=4)) == 1
    assert call(_pool(), scale=0.0) == 1 and call(_pool(), scale=float("nan")) == 1
    assert call(_pool(), pts=info.max_page_blocks - 1) == 1  # page table too narrow
    assert call(_pool(), sts=info.max_stream_blocks - 1) == 1
    assert call(_pool(), q=MIS) == 1 and call(_pool(k=MIS)) == 1   # TMA and vector loads need 16 bytes


def test_append_rejects_malformed_calls(lib):
    call = lambda pool, k=A, v=A, qs=None, qd=None, slots=A, count=4: lib.padoc_append_inputs(
        ctypes.byref(pool) if pool is not None else None, k, v, qs, 10, 16, qd, None, slots, count, None)
    assert call(None) == 1
    assert call(_pool(), count=-1) == 1
    assert call(_pool(), count=0) == 0                      # nothing to do, nothing launched
    assert call(_pool(), k=None) == 1 and call(_pool(), slots=None) == 1
    assert call(_pool(), qs=A, qd=None) == 1                # queries without a destination
    assert call(_pool(d=6, dtype=pa.PADOC_DTYPE_F32)) == 2  # 24-byte rows: no 16-byte vectors
    assert call(_pool(dtype=7)) == 1
    assert call(_pool(), k=MIS) == 1


def test_prefill_rejects_malformed_calls(lib):
    def call(T=100, hq=16, hkv=2, d=128, dtype=pa.PADOC_DTYPE_BF16, scale=0.1, q=A, qt=128, kt=128):
        return lib.padoc_ancestor_prefill_attn(q, A, A, dtype, T, hq, hkv, d, A, A, A, A, qt, kt, scale, A, A, None)
    assert call(T=-1) == 1 and call(hq=16, hkv=3) == 1 and call(scale=-1.0) == 1
    assert call(T=0) == 0
    assert call(q=None) == 1 and call(q=MIS) == 1
    assert call(d=64) == 2                                  # the tensor-core path is head_dim 128
    assert call(dtype=9) == 2
    assert call(qt=64) == 1                                 # the tile map must use the kernel's tiles


def test_prefill_bwd_rejects_malformed_calls(lib):
    (qq, qk), (kq, kk) = pa.padoc_prefill_bwd_tile_shapes(pa.PADOC_DTYPE_BF16, 128)
    qmap = pa.padoc_tile_map_dev(A, A, A, None, qq, qk)
    kmap = pa.padoc_tile_map_dev(A, A, A, A, kq, kk)
    need = pa.padoc_prefill_bwd_workspace_size(100, 16)

    def call(T=100, d=128, dtype=pa.PADOC_DTYPE_BF16, ws=A, wsb=need, qm=qmap, km=kmap, dq=A):
        return lib.padoc_ancestor_prefill_bwd(A, A, A, A, A, A, dtype, T, 16, 2, d, A, ctypes.byref(qm),
                                              ctypes.byref(km), 0.1, dq, A, A, ws, wsb, None)
    assert call(T=-5) == 1 and call(d=64) == 2 and call(dtype=9) == 2
    assert call(T=0) == 0
    assert call(dq=None) == 1 and call(dq=MIS) == 1
    assert call(ws=A + 16) == 1                             # workspace on a 256-byte boundary
    assert call(wsb=need - 1) == 3                          # WORKSPACE_TOO_SMALL
    bad_q = pa.padoc_tile_map_dev(A, A, A, None, qq * 2, qk)
    no_order = pa.padoc_tile_map_dev(A, A, A, None, kq, kk)
    assert call(qm=bad_q) == 1 and call(km=no_order) == 1   # maps built with other tiles / no k-tile order


def test_combine_rejects_malformed_calls(lib):
    call = lambda S=2, R=10, d=128, out=A, po=A, dt=pa.PADOC_DTYPE_BF16: lib.padoc_splitk_combine(
        po, A, S, R, d, dt, out, A, None)
    assert call(S=-1) == 1 and call(R=-1) == 1 and call(d=130) == 1 and call(d=512) == 1
    assert call(R=0) == 0
    assert call(out=None) == 1 and call(po=MIS) == 1


def test_wait_timeout_selftest_rejects_malformed_calls(lib):
    call = lambda limit=1000, site=5, gave_up=A: lib.padoc_selftest_wait_timeout(limit, site, gave_up, None)
    assert call(limit=0) == 1 and call(limit=100001) == 1   # limits outside 1 us .. 0.1 s
    assert call(site=-1) == 1 and call(gave_up=None) == 1


def _pool8(block_size=16, hkv=2, d=128, k=A, v=A, ks=A, vs=A):
    return pa.padoc_kv_pool_e4m3(k, v, ks, vs, 64, block_size, hkv, d)


def test_e4m3_calls_reject_malformed_calls(lib):
    info = _decode_info(lib)
    dec = lambda pool, q=A, ws=1 << 20: lib.padoc_branch_decode_attn_e4m3(
        ctypes.byref(pool) if pool is not None else None, ctypes.byref(info), A, A, 8, A, 8, q, 0.1, A, A, A, ws, None)
    assert dec(None) == 1
    assert dec(_pool8(ks=None)) == 1 and dec(_pool8(k=None)) == 1       # codes and scales are required
    assert dec(_pool8(hkv=4)) == 1 and dec(_pool8(block_size=32)) == 1  # pool and plan disagree
    assert dec(_pool8(k=MIS)) == 1 and dec(_pool8(vs=A + 2)) == 1       # 16-byte codes, 4-byte scales
    assert dec(_pool8(), q=MIS) == 1
    assert dec(_pool8(), ws=16) == 3                                    # workspace below the plan's need
    quant = lambda pool, k=A, v=A, blocks=A, count=3: lib.padoc_quantize_kv_blocks(
        ctypes.byref(pool) if pool is not None else None, k, v, blocks, count, None)
    assert quant(None) == 1 and quant(_pool8(), count=-1) == 1
    assert quant(_pool8(), count=0) == 0                                # nothing to do
    assert quant(_pool8(), blocks=None) == 1 and quant(_pool8(), k=MIS) == 1
    assert quant(_pool8(d=64)) == 2 and quant(_pool8(block_size=8)) == 2
    app = lambda pool, slots=A, qs=None, qd=None, count=4: lib.padoc_append_inputs_e4m3(
        ctypes.byref(pool) if pool is not None else None, A, A, qs, 10, 16, qd, None, slots, count, None)
    assert app(None) == 1 and app(_pool8(), count=-1) == 1
    assert app(_pool8(), count=0) == 0
    assert app(_pool8(), slots=None) == 1 and app(_pool8(), qs=A, qd=None) == 1
    assert app(_pool8(d=64)) == 2


def test_launch_decode_step_rejects_malformed_calls(lib):
    info = _decode_info(lib)
    words = 4096
    call = lambda stage=A, sw=words, opt=2048, pts=8, ost=3072, sts=8, dev=A, dcap=words, qh=A: lib.padoc_launch_decode_step(
        ctypes.byref(_pool()), ctypes.byref(info), stage, sw, opt, pts, ost, sts, dev, dcap, qh, A, 0.1, A, A, A, A, A,
        1 << 20, None, None, None, None, None, None)
    assert call(stage=None) == 1 and call(qh=None) == 1 and call(dev=None) == 1
    assert call(sw=info.plan_ints - 1) == 1                  # the stage must hold the blob
    assert call(dcap=words - 1) == 1                         # the device buffer must hold the stage
    assert call(dev=A + 128) == 1                            # 256-byte aligned device buffer
    assert call(opt=2047) == 1 and call(ost=3073) == 1       # tables on 128-byte boundaries
    assert call(opt=0) == 1                                  # tables after the blob
    assert call(ost=2048) == 1                               # tables must not overlap
    assert call(opt=4064, pts=64) == 1                       # a table past the stage
    piped = lambda ev: lib.padoc_launch_decode_step(ctypes.byref(_pool()), ctypes.byref(info), A, words, 2048, 8, 3072, 8,
                                                    A, words, A, A, 0.1, A, A, A, A, A, 1 << 20, None, A, A, ev, A, A)
    assert piped(None) == 1                                  # copy streams need the three events
