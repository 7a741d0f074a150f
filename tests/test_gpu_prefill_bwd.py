"""GPU parity of the prefill backward: dQ, dK, dV of the CUDA path through the C ABI against the
fp64 oracle's gradients, on the same seeded inputs, with O and lse from the CUDA forward.

Tolerance, from the arithmetic of the bf16 path: Q, K, V, dO and O are bf16 inputs; S, dP and the
accumulators are fp32; P and dS enter the accumulating MMAs rounded to bf16 and dQ, dK, dV are
stored in bf16, each a relative rounding of 2^-9 on terms of mixed sign, and D = dO.O uses the
forward's bf16 O. Per row of each gradient (a token's head_dim x heads values) the error stays
within a few units of 2^-9 of the row's largest value, so the check is
|got - ref| <= 2^-6 * rowmax|ref| + 2^-8 * rms(ref) elementwise; the second term covers rows whose
values are small against the tensor. The fp32 bring-up path (fp32 FMA throughout) is held to
1e-4 of the same scales.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import inputs
from paper_2608_06146_gb300 import padoc_attn as pa
from paper_2608_06146_gb300.engine import PrefillBwdPlan, PrefillPlan
from paper_2608_06146_gb300.inputs import PageSpec, Workload

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
BF16_RTOL, BF16_ATOL = 2.0 ** -6, 2.0 ** -8
F32_RTOL, F32_ATOL = 1e-4, 1e-5


@pytest.fixture(scope="module", autouse=True)
def _build():
    pbuild.build()
    pa.load_library()


def run_bwd(wl: Workload, seed: int, scale_in=1.0, q_rows=None, k_rows=None, repeat=1):
    q, k, v = inputs.packed_qkv(wl, seed, scale_in)
    g = inputs.packed_dout(wl, seed)
    scale = 1.0 / math.sqrt(wl.head_dim)
    T, Hq, Hkv, d = q.shape[0], wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    qd, kd, vd, gd = (x.to(DEV) for x in (q, k, v, g))
    fwd = PrefillPlan(wl.pages, wl.dtype, d, DEV)
    out = torch.empty((T, Hq, d), dtype=wl.dtype, device=DEV)
    lse = torch.empty((T, Hq), dtype=torch.float32, device=DEV)
    fwd.run(qd, kd, vd, scale, out, lse)
    bwd = PrefillBwdPlan(wl.pages, wl.dtype, d, Hq, DEV)
    runs = []
    for _ in range(repeat):
        dq = torch.full((T, Hq, d), float("nan"), dtype=wl.dtype, device=DEV)
        dk = torch.full((T, Hkv, d), float("nan"), dtype=wl.dtype, device=DEV)
        dv = torch.full((T, Hkv, d), float("nan"), dtype=wl.dtype, device=DEV)
        bwd.run(qd, kd, vd, out, gd, lse, scale, dq, dk, dv)
        pa.padoc_check_device_errors()
        runs.append(tuple(x.float().cpu().numpy() for x in (dq, dk, dv)))
    ref = oracle.prefill_bwd(wl.pages, q, k, v, g, scale, q_rows, k_rows)
    qs = slice(None) if q_rows is None else np.asarray(q_rows)
    ks = slice(None) if k_rows is None else np.asarray(k_rows)
    got = [(a[qs], b[ks], c[ks]) for a, b, c in runs]
    return got, ref


def assert_grad_close(got, ref, dtype, name):
    rtol, atol = (BF16_RTOL, BF16_ATOL) if dtype == torch.bfloat16 else (F32_RTOL, F32_ATOL)
    assert np.isfinite(got).all(), f"{name}: non-finite values"
    rows = ref.reshape(ref.shape[0], -1)
    err = np.abs(got.reshape(rows.shape) - rows)
    bound = rtol * np.abs(rows).max(1, keepdims=True) + atol * math.sqrt(float((rows ** 2).mean()))
    bad = err > bound
    if bad.any():
        r = int(np.argmax((err / bound).max(1)))
        raise AssertionError(f"{name}: {int(bad.sum())} of {bad.size} values out of bound; worst row {r}: "
                             f"max err {err[r].max():.3e}, bound {bound[r, 0]:.3e}, row max {np.abs(rows[r]).max():.3e}")


def check(wl, seed, **kw):
    got, ref = run_bwd(wl, seed, **kw)
    for (a, b, c) in got:
        assert_grad_close(a, ref[0], wl.dtype, "dQ")
        assert_grad_close(b, ref[1], wl.dtype, "dK")
        assert_grad_close(c, ref[2], wl.dtype, "dV")
    return got


def test_prefill_bwd_tiny_fp32():
    check(inputs.tiny_page(), 0, scale_in=1 / 8)


def test_prefill_bwd_bf16_multi_page_ragged():
    # several tiles per page, pages not aligned to 64 or 128, a ragged last tile, shuffled forks,
    # a one-token branch, a page that is one causal stream
    pages = [PageSpec(300, 40, [8, 40, 16, 0, 24], [50, 1, 77, 130, 9]),
             PageSpec(129, 0, [0, 0], [3, 200]),
             PageSpec(5, 16, [16], [1]),
             PageSpec(257, 64, [], [])]
    check(Workload("ragged", pages, 16, 2, 128, torch.bfloat16, "prefill"), 6)


@pytest.mark.parametrize("hq,hkv", [(8, 8), (4, 1), (6, 2), (16, 2)])
def test_prefill_bwd_bf16_gqa_groups(hq, hkv):
    # every query head of a KV head's group adds into that KV head's dK and dV
    pages = [PageSpec(200, 16, [8, 16, 4], [40, 30, 60])]
    check(Workload("gqa", pages, hq, hkv, 128, torch.bfloat16, "prefill"), 7)


def test_prefill_bwd_bf16_edge_pages():
    # fewer tokens than one step (T < 64), a one-token page, a page with P = 0, f_k = 0 and f_k = L
    for pages in ([PageSpec(20, 8, [0, 8, 3], [5, 1, 9])],
                  [PageSpec(1, 0, [], []), PageSpec(0, 7, [0, 7], [64, 65]), PageSpec(63, 1, [1], [1])]):
        check(Workload("edge", pages, 16, 2, 128, torch.bfloat16, "prefill"), 8)


def test_prefill_bwd_bf16_deterministic():
    # no atomics: two calls give bit-identical gradients
    pages = [PageSpec(300, 24, [8, 16, 24], [100, 3, 250])]
    got = check(Workload("det", pages, 16, 2, 128, torch.bfloat16, "prefill"), 9, repeat=2)
    for a, b in zip(got[0], got[1]):
        np.testing.assert_array_equal(a, b)


def _sample_rows(wl, rng, n_per_page, pages):
    rows, base = [], 0
    for p, pg in enumerate(wl.pages):
        S = pg.packed_len
        if p in pages:
            M = pg.prefix_len + pg.layout_len
            fixed = [0, 1, pg.prefix_len - 1, M - 1, M, S - 1] if M else [0, S - 1]
            pick = set(x for x in fixed if 0 <= x < S) | set(int(x) for x in rng.integers(0, S, n_per_page))
            rows += [base + x for x in sorted(pick)]
        base += S
    return rows


def test_prefill_bwd_bf16_packed_full_size_sampled():
    # 8 pages x 4096 tokens through the full CUDA path; sampled dQ rows of every page and sampled
    # dK/dV rows (prefix starts, the stream's end, branch tokens) of the first and last page
    wl = inputs.packed_prefill()
    rng = np.random.default_rng(40)
    q_rows = _sample_rows(wl, rng, 24, range(len(wl.pages)))
    k_rows = _sample_rows(wl, rng, 40, [0, len(wl.pages) - 1])
    check(wl, 4, q_rows=q_rows, k_rows=k_rows)


def test_prefill_bwd_bf16_shuffled_branches_sampled():
    wl = inputs.packed_prefill(seed=5, num_pages=2, shuffle_branches=True)
    rng = np.random.default_rng(41)
    check(wl, 5, q_rows=_sample_rows(wl, rng, 60, [0, 1]), k_rows=_sample_rows(wl, rng, 60, [1]))
