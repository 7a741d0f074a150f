"""Benchmark of padoc_attn on one GB300 (or N independent GPUs, weak scaling).

A step is one pass of the hot path over one batch:
  decode  -- one decode step for every branch of the 32-page concurrent serving batch (prefix
             uniform in [1024,4096], Poisson(20) branches per page, log-normal private lengths):
             the decode plan's split-K kernel over the paged bf16 cache plus the split-K merge;
  prefill -- the packed ancestor prefill of 8 pages x 4096 tokens (reported in "prefill");
  prefill_bwd -- its gradients dQ, dK, dV for a seeded upstream gradient (reported in
             "prefill_bwd");
  chunk_prefill -- branch prefill over the paged cache of the serving batch's pages, every branch
             as one chunk (reported in "branch_prefill");
  loop    -- Algorithm 1 over the serving batch's 32 pages, from admission to the last EOS
             (reported in "loop": end to end through the engine, and the device time of the same
             steps replayed from a CUDA graph).
Headline metric: decode queries/s (one query = one branch's newest token, all 16 query heads).

Timing: W untimed warm-up steps, then K steps between CUDA events on the launching stream, with
a barrier and a synchronize on both sides; the max over ranks is reported. Decode rotates over
input replicas in distinct memory whose total exceeds 4x L2, so no step reads a previous step's
data from L2. Prefill flushes L2 between steps (a write of a buffer larger than L2) and times
each step with its own events. nvidia-smi samples clocks during the timed region.

--impl reference times the fp64 CPU oracle on the host cores on a bounded sample of the same
decode workload (the paper has no code; the oracle is the reference program here).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "ancestor-attn decode queries/s, % of HBM roofline; packed prefill TFLOP/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# DRAM traffic per launch, dram__bytes_read.sum + dram__bytes_write.sum, copied from one ncu capture
# of each kernel as it stands; None where no capture of the current kernel exists. Decode: one step =
# its kernels' counters added up (bf16: the decode grid and the merge, captured with the caches left
# as the pipeline leaves them, so that the merge reads its partials from L2 as it does in the timed
# step, the mean of two consecutive steps; E4M3: the tensor-core grid, the warp grid and the merge,
# cold caches). Prefill: cold caches. Prefill backward: both passes and the merge of the split key
# tiles, cold caches.
TRAFFIC_BYTES = {"decode": 201_274_880,
                 "decode_e4m3": 114_668_800,
                 "prefill": 260_600_000,
                 "prefill_bwd": 1_670_324_480}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


class ClockSampler:
    """nvidia-smi clock/throttle sampling in the background during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(prefix="clocks", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), float(parts[3]) if parts[3] not in ("[N/A]", "N/A") else 0.0,
                             parts[5], parts[6], parts[7], parts[8]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        loaded = [r for r in rows if r[2] > 0.3 * max(x[2] for x in rows)] or rows
        reasons = set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            for n, v in zip(names, r[3:]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(r[0] for r in loaded), "sm_max_mhz": max(r[1] for r in rows),
                "samples": len(rows), "reasons": sorted(reasons)}


# ------------------------------------------------------------------------------------------------
# Workloads
# ------------------------------------------------------------------------------------------------

def decode_bytes(wl, layout_streams=False, kv_bytes=2, scale_bytes=0):
    """Minimum HBM bytes of one decode step: each page's shared stream once per KV head up to the
    last row any of its streams sees (P + max f_k, or P + L when the layout stream is decoded),
    every private row once, Q in, O and LSE out. ``kv_bytes`` per K/V element; ``scale_bytes`` per
    (16-token block, KV head) for K and for V each (a quantized cache's scales)."""
    Hq, Hkv, d = wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    shared = priv = S = sblk = 0
    for pg in wl.pages:
        n = pg.num_branches + (1 if layout_streams else 0)
        if n == 0:
            continue
        cut = pg.prefix_len + (pg.layout_len if layout_streams else max(pg.fork_offset))
        shared += cut
        priv += int(sum(pg.branch_len))
        sblk += -(-cut // 16) + sum(-(-b // 16) for b in pg.branch_len)
        S += n
    return ((shared + priv) * Hkv * d * 2 * kv_bytes + sblk * Hkv * 2 * scale_bytes
            + S * Hq * d * 2 * 2 + S * Hq * 4)


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


def prefill_flops(wl):
    return 4.0 * wl.head_dim * wl.num_q_heads * visible_pairs(wl.pages)


def l2_bytes(torch):
    try:
        return int(torch.cuda.get_device_properties(torch.cuda.current_device()).L2_cache_size)
    except Exception:
        return 129 * 1024 * 1024


class StepGraphs:
    """Decode steps captured in CUDA graphs: graph g holds ``n`` consecutive steps starting at step
    ``first``. A step's kernels are programmatic dependents of the previous step's, and capture keeps
    those dependencies as programmatic edges, so consecutive steps inside a graph overlap exactly as
    they do when launched one by one; what the graph removes is the host's per-launch cost."""

    def __init__(self, torch, step, first, n, stream):
        self.g = torch.cuda.CUDAGraph()
        cap = torch.cuda.Stream()
        cap.wait_stream(stream)
        with torch.cuda.graph(self.g, stream=cap):
            s = torch.cuda.current_stream()
            for i in range(n):
                step(first + i, s)
        stream.wait_stream(cap)
        self.n = n

    def replay(self):
        self.g.replay()


def time_steps(args, torch, world, stream, step, steady=True, steady_steps=25000, steady_graph=1000):
    """W eager warm-up steps, then the graphs are captured and uploaded. Inside the clock sampler:
    a long run of back-to-back steps (``steady_steps``, replays of a ``steady_graph``-step graph,
    each replay between its own CUDA events; median, minimum and maximum per step), and right after
    it, with no idle gap, exactly K steps from CUDA graphs between one pair of CUDA events,
    bracketed by a barrier and a synchronize. The long run comes first so that the K steps are
    measured at the clocks the GPU holds under this load, not while it ramps up from idle. With
    --no-steady the long-run graph is replayed once, untimed, instead."""
    import paper_2608_06146_gb300.padoc_attn as pa
    for i in range(args.warmup):
        step(i, stream)
    torch.cuda.synchronize()
    pa.padoc_check_device_errors(stream)
    K = args.steps
    G = min(K, 500)
    graphs = [StepGraphs(torch, step, args.warmup, G, stream)]
    if K % G:
        graphs.append(StepGraphs(torch, step, args.warmup + (K // G) * G, K % G, stream))
    timed = [graphs[0]] * (K // G) + graphs[1:]
    sg = StepGraphs(torch, step, args.warmup, steady_graph, stream)
    for g in graphs + [sg]:    # first replays upload the graphs
        g.replay()
    torch.cuda.synchronize()
    pa.padoc_check_device_errors(stream)
    reps = max(1, steady_steps // steady_graph) if (steady and not args.no_steady) else 0
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    res = {}
    with ClockSampler(physical_gpu_index(torch.cuda.current_device())) as clk:
        barrier(torch, world)
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            sg.replay()
            for a, b in evs:
                a.record(stream)
                sg.replay()
                b.record(stream)
            ev0.record(stream)
            for g in timed:
                g.replay()
            ev1.record(stream)
        torch.cuda.synchronize()
        barrier(torch, world)
    res["ms"] = ev0.elapsed_time(ev1) / K
    if reps:
        per = sorted(a.elapsed_time(b) / steady_graph for a, b in evs)
        res["steady"] = dict(steps=reps * steady_graph, graph_steps=steady_graph, replays=reps,
                             median_ms=statistics.median(per), min_ms=per[0], max_ms=per[-1],
                             mean_ms=sum(per) / len(per))
    pa.padoc_check_device_errors(stream)
    res["clocks"] = clk.summary()
    return res


def bench_decode(args, torch, dev, rank, world, layout_streams=False):
    """The serving-batch decode step (with ``layout_streams``, every page's layout stream is decoded
    too, as Algorithm 1 decodes every live stream)."""
    from paper_2608_06146_gb300 import inputs
    from paper_2608_06146_gb300 import padoc_attn as pa
    from paper_2608_06146_gb300.engine import DecodePlan

    wl = inputs.serving_batch(seed=3 + 1000 * rank)
    scale = 1.0 / math.sqrt(wl.head_dim)
    di = inputs.decode_inputs(wl, 3 + 1000 * rank, pool_slack=1.0, layout_streams=layout_streams)
    plan = DecodePlan(wl.pages, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, dev, tc_ctas=args.tc_ctas,
                      warp_ctas=args.warp_ctas, split_tokens=args.split_tokens, layout_streams=layout_streams)
    S = plan.num_streams
    per_replica = (di.k_pool.numel() + di.v_pool.numel()) * 2
    R = args.replicas if args.replicas > 0 else max(2, math.ceil(4 * l2_bytes(torch) / per_replica) + 1)
    k_pools = [di.k_pool.to(dev) for _ in range(R)]
    v_pools = [di.v_pool.to(dev) for _ in range(R)]
    qs = [di.q.to(dev) for _ in range(R)]
    page_table = torch.from_numpy(di.page_table).to(dev)
    stream_table = torch.from_numpy(di.stream_table).to(dev)
    outs = [torch.empty((S, wl.num_q_heads, wl.head_dim), dtype=torch.bfloat16, device=dev) for _ in range(R)]
    lses = [torch.empty((S, wl.num_q_heads), dtype=torch.float32, device=dev) for _ in range(R)]
    stream = torch.cuda.current_stream()

    def step(i, s):
        r = i % R
        plan.run(k_pools[r], v_pools[r], page_table, stream_table, qs[r], scale, outs[r], lses[r], s)

    timing = time_steps(args, torch, world, stream, step, steady=not layout_streams)
    nbytes = decode_bytes(wl, layout_streams)
    info = plan.info
    launches = (1 if info.num_tc_items > 0 or info.num_warps > 0 else 0) + 1   # the decode grid + the merge
    res = dict(ms=timing["ms"], streams=S, bytes=nbytes, launches=launches, clocks=timing["clocks"], replicas=R,
               pages=len(wl.pages), e2e_ms=None, h2d=0, d2h=0, steady=timing.get("steady"))
    if args.no_e2e or layout_streams:
        return res

    # end to end through the public API, every step: the plan brought to the step's lengths
    # (padoc_advance_decode_plan, which checks and patches the host plan in place; this batch's
    # lengths do not change from step to step, so nothing moves), and one library call that copies
    # the step's integers (plan blob, page and stream block tables) and queries from pinned host
    # memory to the device, decodes, and copies O and LSE back to pinned host memory. Two buffer
    # sets used in turn and two copy streams: a step's copies in overlap the previous step's decode,
    # its copies out the next step's (the library orders them with the set's events).
    PT, STW = di.page_table.shape[1], di.stream_table.shape[1]
    align = lambda n: (n + 31) // 32 * 32
    plan_ints = int(plan.info.plan_ints)
    off_pt = align(plan_ints)
    off_st = off_pt + align(len(wl.pages) * PT)
    words = off_st + align(S * STW)
    copy_in, copy_out = torch.cuda.Stream(), torch.cuda.Stream()
    sets = []
    for _ in range(2):
        stage = torch.zeros(words, dtype=torch.int32).pin_memory()
        h = stage.numpy()
        h[:plan_ints] = plan.plan_host
        h[off_pt:off_pt + len(wl.pages) * PT] = di.page_table.reshape(-1)
        h[off_st:off_st + S * STW] = di.stream_table.reshape(-1)
        evs = [torch.cuda.Event() for _ in range(3)]
        for e in evs:            # created (and ev_free set) before the first step
            e.record(stream)
        sets.append(dict(stage=stage, info=pa.padoc_decode_plan.from_buffer_copy(plan.info),
                         dev_ints=torch.empty(words, dtype=torch.int32, device=dev),
                         q_host=di.q.pin_memory(), q_dev=torch.empty_like(qs[0]),
                         out=torch.empty_like(outs[0]), lse=torch.empty_like(lses[0]),
                         o_host=torch.empty((S, wl.num_q_heads, wl.head_dim), dtype=torch.bfloat16).pin_memory(),
                         l_host=torch.empty((S, wl.num_q_heads), dtype=torch.float32).pin_memory(), ev=evs))
    ws2 = [plan.workspace, torch.empty_like(plan.workspace)]
    lens = np.ascontiguousarray(plan.plan_host[plan.info.off_private_len:plan.info.off_private_len + S])
    # one pa.DecodeStep per (buffer set, input replica): the arguments are marshalled once, as a caller
    # with a fixed pool does
    calls = [[pa.DecodeStep(k_pools[r], v_pools[r], st_["info"], st_["stage"], words, plan_ints, off_pt, PT, off_st,
                            STW, st_["dev_ints"], st_["q_host"], st_["q_dev"], scale, st_["out"], st_["lse"],
                            st_["o_host"], st_["l_host"], ws2[b], lens, stream, copy_in, copy_out, st_["ev"][0],
                            st_["ev"][1], st_["ev"][2]) for r in range(R)] for b, st_ in enumerate(sets)]

    def e2e_step(i):
        b = i & 1
        sets[b]["ev"][1].synchronize()     # this set's previous copies in have run: its stage may change
        if not calls[b][i % R]():
            raise RuntimeError("plan advance refused")

    for i in range(max(args.warmup, 2)):
        e2e_step(i)
    torch.cuda.synchronize()
    barrier(torch, world)
    t0 = time.perf_counter()
    e2e_steps = min(args.steps, 2000)
    for i in range(e2e_steps):
        e2e_step(i)
    torch.cuda.synchronize()
    e2e_ms = (time.perf_counter() - t0) * 1e3 / e2e_steps
    barrier(torch, world)
    h2d = words * 4 + sets[0]["q_host"].numel() * 2
    d2h = sets[0]["o_host"].numel() * 2 + sets[0]["l_host"].numel() * 4
    res.update(e2e_ms=e2e_ms, h2d=h2d, d2h=d2h)
    return res


def bench_decode_replicas(args, torch, dev, rank, world, shape):
    """A decode step over R replicas of one page shape, decoded together (one decode call per step):
    ``shape`` "decode_page" (P = 2048, L = 256, 16 branches) or "dense_page" (P = 4096, L = 512,
    64 branches); each replica has its own seeded K/V/Q in distinct memory, R chosen so that the
    batch's cache exceeds 4x L2 (every step reads the whole batch, so no step is served from L2)."""
    from paper_2608_06146_gb300 import inputs
    from paper_2608_06146_gb300 import padoc_attn as pa
    from paper_2608_06146_gb300.engine import DecodePlan

    base = inputs.WORKLOADS[shape](seed=1 if shape == "decode_page" else 2)
    pg = base.pages[0]
    page_bytes = (pg.stream_len + sum(pg.branch_len)) * base.num_kv_heads * base.head_dim * 2 * 2
    R = math.ceil(4 * l2_bytes(torch) / page_bytes) + 1
    wl = inputs.Workload(f"{R} x {shape}", [pg] * R, base.num_q_heads, base.num_kv_heads, base.head_dim,
                         base.dtype, "decode")
    seed = 7 + 1000 * rank
    di = inputs.decode_inputs(wl, seed, pool_slack=1.0)
    plan = DecodePlan(wl.pages, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, dev, tc_ctas=args.tc_ctas,
                      warp_ctas=args.warp_ctas, split_tokens=args.split_tokens)
    S = plan.num_streams
    k_pool, v_pool, q = di.k_pool.to(dev), di.v_pool.to(dev), di.q.to(dev)
    page_table = torch.from_numpy(di.page_table).to(dev)
    stream_table = torch.from_numpy(di.stream_table).to(dev)
    out = torch.empty((S, wl.num_q_heads, wl.head_dim), dtype=torch.bfloat16, device=dev)
    lse = torch.empty((S, wl.num_q_heads), dtype=torch.float32, device=dev)
    scale = 1.0 / math.sqrt(wl.head_dim)
    stream = torch.cuda.current_stream()

    def step(i, s):
        plan.run(k_pool, v_pool, page_table, stream_table, q, scale, out, lse, s)

    timing = time_steps(args, torch, world, stream, step, steady=False)
    info = plan.info
    launches = (1 if info.num_tc_items > 0 or info.num_warps > 0 else 0) + 1
    return dict(ms=timing["ms"], streams=S, pages=R, bytes=decode_bytes(wl), launches=launches,
                clocks=timing["clocks"], tc_items=int(info.num_tc_items), warp_items=int(info.num_items - info.num_tc_items))


def bench_decode_e4m3(args, torch, dev, rank, world):
    """The serving-batch decode step over the FP8 (E4M3) cache: the same pages, plan and queries, the
    pool quantized from the bf16 one (whole blocks) in R replicas in distinct memory."""
    from paper_2608_06146_gb300 import inputs
    from paper_2608_06146_gb300 import padoc_attn as pa
    from paper_2608_06146_gb300.engine import DecodePlan

    wl = inputs.serving_batch(seed=3 + 1000 * rank)
    scale = 1.0 / math.sqrt(wl.head_dim)
    di = inputs.decode_inputs(wl, 3 + 1000 * rank, pool_slack=1.0)
    plan = DecodePlan(wl.pages, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, dev, tc_ctas=args.tc_ctas,
                      warp_ctas=args.warp_ctas, split_tokens=args.split_tokens)
    S = plan.num_streams
    per_replica = di.k_pool.numel() * 2 + di.num_blocks * wl.num_kv_heads * 8
    R = max(2, math.ceil(4 * l2_bytes(torch) / per_replica) + 1)
    k_bf, v_bf = di.k_pool.to(dev), di.v_pool.to(dev)
    blocks = torch.arange(di.num_blocks, dtype=torch.int32, device=dev)
    pools = []
    for _ in range(R):
        pool = pa.E4M3Pool(di.num_blocks, wl.num_kv_heads, wl.head_dim, dev)
        pa.padoc_quantize_kv_blocks(pool, k_bf, v_bf, blocks)
        pools.append(pool)
    del k_bf, v_bf
    qs = [di.q.to(dev) for _ in range(R)]
    page_table = torch.from_numpy(di.page_table).to(dev)
    stream_table = torch.from_numpy(di.stream_table).to(dev)
    outs = [torch.empty((S, wl.num_q_heads, wl.head_dim), dtype=torch.bfloat16, device=dev) for _ in range(R)]
    lses = [torch.empty((S, wl.num_q_heads), dtype=torch.float32, device=dev) for _ in range(R)]
    stream = torch.cuda.current_stream()

    def step(i, s):
        r = i % R
        pa.padoc_branch_decode_attn_e4m3(pools[r], plan.info, plan.plan_dev, page_table, stream_table, qs[r], scale,
                                         outs[r], lses[r], plan.workspace, s)

    timing = time_steps(args, torch, world, stream, step, steady=False)
    info = plan.info
    # the tensor-core grid, the warp grid (the E4M3 pool runs them apart) and the merge
    launches = (1 if info.num_tc_items > 0 else 0) + (1 if info.num_warps > 0 else 0) + 1
    return dict(ms=timing["ms"], streams=S, bytes=decode_bytes(wl, kv_bytes=1, scale_bytes=4), launches=launches,
                clocks=timing["clocks"], replicas=R)


def bench_prefill(args, torch, dev, rank, world, shuffle=False):
    """The packed prefill of 8 pages x 4096 tokens (with ``shuffle``, each page's branches permuted
    so that the fork offsets are not monotone in the branch index)."""
    from paper_2608_06146_gb300 import inputs
    from paper_2608_06146_gb300 import padoc_attn as pa
    from paper_2608_06146_gb300.engine import PrefillPlan

    wl = inputs.packed_prefill(seed=4 + 1000 * rank, shuffle_branches=shuffle)
    q, k, v = inputs.packed_qkv(wl, 4 + 1000 * rank)
    plan = PrefillPlan(wl.pages, wl.dtype, wl.head_dim, dev)
    q, k, v = q.to(dev), k.to(dev), v.to(dev)
    out = torch.empty(q.shape, dtype=q.dtype, device=dev)
    lse = torch.empty(q.shape[:2], dtype=torch.float32, device=dev)
    scale = 1.0 / math.sqrt(wl.head_dim)
    flush = torch.empty(2 * l2_bytes(torch), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    steps = max(3, min(args.steps, 20))
    for _ in range(max(args.warmup, 3)):
        plan.run(q, k, v, scale, out, lse, stream)
    pa.padoc_check_device_errors(stream)
    barrier(torch, world)
    times = []
    for _ in range(steps):
        flush.fill_(1)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        plan.run(q, k, v, scale, out, lse, stream)
        e1.record(stream)
        e1.synchronize()
        times.append(e0.elapsed_time(e1))
    pa.padoc_check_device_errors(stream)
    barrier(torch, world)
    ms = sum(times) / len(times)
    return dict(ms=ms, flops=prefill_flops(wl), tokens=plan.T, steps=steps)


def bench_prefill_bwd(args, torch, dev, rank, world):
    """The gradients of the packed prefill (dQ, dK, dV) for a seeded upstream gradient, after one
    forward that supplies O and lse; each timed step is one padoc_ancestor_prefill_bwd call."""
    from paper_2608_06146_gb300 import inputs
    from paper_2608_06146_gb300 import padoc_attn as pa
    from paper_2608_06146_gb300.engine import PrefillBwdPlan, PrefillPlan

    wl = inputs.packed_prefill(seed=4 + 1000 * rank)
    q, k, v = (x.to(dev) for x in inputs.packed_qkv(wl, 4 + 1000 * rank))
    g = inputs.packed_dout(wl, 4 + 1000 * rank).to(dev)
    scale = 1.0 / math.sqrt(wl.head_dim)
    fwd = PrefillPlan(wl.pages, wl.dtype, wl.head_dim, dev)
    out = torch.empty(q.shape, dtype=q.dtype, device=dev)
    lse = torch.empty(q.shape[:2], dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    fwd.run(q, k, v, scale, out, lse, stream)
    plan = PrefillBwdPlan(wl.pages, wl.dtype, wl.head_dim, wl.num_q_heads, dev)
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    flush = torch.empty(2 * l2_bytes(torch), dtype=torch.uint8, device=dev)
    steps = max(3, min(args.steps, 20))
    for _ in range(max(args.warmup, 3)):
        plan.run(q, k, v, out, g, lse, scale, dq, dk, dv, stream)
    pa.padoc_check_device_errors(stream)
    barrier(torch, world)
    times = []
    for _ in range(steps):
        flush.fill_(1)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        plan.run(q, k, v, out, g, lse, scale, dq, dk, dv, stream)
        e1.record(stream)
        e1.synchronize()
        times.append(e0.elapsed_time(e1))
    pa.padoc_check_device_errors(stream)
    barrier(torch, world)
    ms = sum(times) / len(times)
    # five T x T x d products per visible pair (S, dP, dV, dK, dQ): 2.5x the forward's two
    return dict(ms=ms, flops=2.5 * prefill_flops(wl), tokens=plan.T, steps=steps)


def bench_chunk_prefill(args, torch, dev, rank, world):
    """Branch prefill over the paged cache of the 32 serving-batch pages: every branch's tokens as one
    chunk from its branch-initialization token (private rows 0 .. n_k - 1 against the page's shared
    stream up to P + f_k) and every page's layout stream as one shared-stream chunk; each timed step
    is one decode-kernel pass over the chunk plan, with L2 flushed between steps."""
    from paper_2608_06146_gb300 import inputs
    from paper_2608_06146_gb300 import padoc_attn as pa
    from paper_2608_06146_gb300.engine import ChunkPrefillPlan

    seed = 3 + 1000 * rank
    wl = inputs.serving_batch(seed=seed)
    di = inputs.decode_inputs(wl, seed, pool_slack=1.0)
    chunks, table, b = [], [], 0
    pairs = 0
    for p, pg in enumerate(wl.pages):
        for f, n in zip(pg.fork_offset, pg.branch_len):
            chunks.append((p, pg.prefix_len + f, 0, n))
            table.append(di.stream_table[b])
            b += 1
            pairs += n * (pg.prefix_len + f) + n * (n + 1) // 2
        chunks.append((p, pg.prefix_len, -1, pg.layout_len))
        table.append(np.full(di.stream_table.shape[1], -1, np.int32))
        pairs += pg.layout_len * pg.prefix_len + pg.layout_len * (pg.layout_len + 1) // 2
    page_len = np.array([pg.stream_len for pg in wl.pages], np.int32)
    plan = ChunkPrefillPlan(page_len, chunks, np.stack(table), wl.num_q_heads, wl.num_kv_heads, wl.head_dim, dev,
                            tc_ctas=args.tc_ctas, warp_ctas=args.warp_ctas)
    T = plan.num_tokens
    q = inputs.randn((T, wl.num_q_heads, wl.head_dim), wl.dtype, seed * 1000 + 98).to(dev)
    out = torch.empty_like(q)
    lse = torch.empty((T, wl.num_q_heads), dtype=torch.float32, device=dev)
    k_pool, v_pool = di.k_pool.to(dev), di.v_pool.to(dev)
    page_table = torch.from_numpy(di.page_table).to(dev)
    scale = 1.0 / math.sqrt(wl.head_dim)
    flush = torch.empty(2 * l2_bytes(torch), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    steps = max(3, min(args.steps, 20))
    for _ in range(max(args.warmup, 3)):
        plan.run(k_pool, v_pool, page_table, q, scale, out, lse, stream)
    pa.padoc_check_device_errors(stream)
    barrier(torch, world)
    times = []
    for _ in range(steps):
        flush.fill_(1)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        plan.run(k_pool, v_pool, page_table, q, scale, out, lse, stream)
        e1.record(stream)
        e1.synchronize()
        times.append(e0.elapsed_time(e1))
    pa.padoc_check_device_errors(stream)
    barrier(torch, world)
    info = plan.info
    return dict(ms=sum(times) / len(times), flops=4.0 * wl.head_dim * wl.num_q_heads * pairs, tokens=T, steps=steps,
                chunks=len(chunks), tc_items=int(info.num_tc_items), warp_items=int(info.num_items - info.num_tc_items))


def bench_loop(args, torch, dev, rank, world):
    """Algorithm 1 over the serving batch's 32 pages: every page is admitted (its prefix K/V appended
    into the pool, untimed), then the loop runs every layout stream and branch from its first input
    to its EOS. Timed twice: (a) end to end through the engine, as a caller runs it (per step one
    library call, padoc_mpd_runner_step: the host scheduler and planner, one host->device copy and
    the append + decode launches; then the step's events handed to the scheduler, padoc_mpd_end_step;
    the inputs' source rows in a table by stream id); the synthetic token source stands in for the
    decoder's sampled outputs, and its events depend only on the pages and the scheduler's stream
    order, so they are drawn once, before the timed region (a warm-up pass records each step's
    stream ids, source rows, forks and EOS flags; the timed pass replays them and checks that the
    scheduler hands out the same stream ids); no step waits for the device; (b) the device work
    alone: the same steps' launches, captured once in a CUDA graph from per-step inputs already on
    the device, replayed."""
    from paper_2608_06146_gb300 import inputs
    from paper_2608_06146_gb300 import padoc_attn as pa
    from paper_2608_06146_gb300.engine import MaskedParallelLoop

    seed = 3 + 1000 * rank
    wl = inputs.serving_batch(seed=seed)
    q, k, v = inputs.packed_qkv(wl, seed)
    qd, kd, vd = q.to(dev), k.to(dev), v.to(dev)
    Hq, Hkv, d = wl.num_q_heads, wl.num_kv_heads, wl.head_dim
    scale = 1.0 / math.sqrt(d)
    nb = sum(-(-(pg.prefix_len + pg.layout_len) // 16) + sum(-(-n // 16) for n in pg.branch_len) for pg in wl.pages) + 64
    order = np.random.default_rng(seed + 77).permutation(nb).astype(np.int32)
    stream = torch.cuda.current_stream()

    def admit_all():
        src = inputs.LoopTokenSource(wl.pages)
        loop = MaskedParallelLoop(nb, Hq, Hkv, d, wl.dtype, dev, block_order=order, tc_ctas=args.tc_ctas,
                                  warp_ctas=args.warp_ctas, split_tokens=args.split_tokens)
        for p in range(len(wl.pages)):
            P, nf, leos, rows = src.admission(p)
            _, new = loop.add_page(P, nf, leos, kd, vd, rows)
            src.admitted(p, new)
        return src, loop

    def run(record):
        src, loop = admit_all()
        torch.cuda.synchronize()
        steps = toks = h2d = 0
        rec, traj = [], []
        t0 = time.perf_counter()
        while loop.status()[1] > 0:
            rows_now = []
            ids, out, lse = loop.step(kd, vd, qd, lambda x: rows_now.append(src.rows(x)) or rows_now[0], scale)
            steps += 1
            toks += len(ids)
            h2d += loop.h2d_bytes
            if record:
                stp = loop.last_step
                rec.append((loop.last_stage[:int(stp.upload_words)].copy(), stp))
            nf, eos = src.events(ids)
            traj.append((ids.copy(), np.asarray(rows_now[0], np.int32).copy(), nf.copy(), eos.copy()))
            src.forked(ids, nf, loop.end_step(nf, eos))
        torch.cuda.synchronize()
        return time.perf_counter() - t0, steps, toks, h2d, rec, traj

    def run_replay(traj):
        _, loop = admit_all()
        cmax = max(len(t[0]) for t in traj)
        n_ids = max(int(t[0].max()) for t in traj if len(t[0])) + 1
        outs_ = [torch.empty((cmax, Hq, d), dtype=wl.dtype, device=dev) for _ in range(2)]
        lses_ = [torch.empty((cmax, Hq), dtype=torch.float32, device=dev) for _ in range(2)]
        row_of = np.zeros(n_ids, np.int32)   # each live stream's source row, by stream id
        # the ids each step hands out, kept for the check after the timed region
        got = np.full(sum(len(t[0]) for t in traj), -1, np.int32)
        counts = np.zeros(len(traj), np.int64)
        torch.cuda.synchronize()
        toks = h2d = 0
        t0 = time.perf_counter()
        for i, (ids_r, rows_r, nf_r, eos_r) in enumerate(traj):
            row_of[ids_r] = rows_r
            C, ids = loop.run_step(kd, vd, qd, row_of, scale, outs_[i & 1], lses_[i & 1])
            if toks + C <= got.size:
                got[toks:toks + C] = ids
            counts[i] = C
            toks += C
            h2d += loop.h2d_bytes
            loop.end_step(nf_r, eos_r)
        torch.cuda.synchronize()
        el = time.perf_counter() - t0
        want = np.concatenate([t[0] for t in traj]) if traj else got
        same = np.array_equal(counts, [len(t[0]) for t in traj]) and np.array_equal(got, want)
        if not same or loop.status()[1] != 0:
            raise RuntimeError("the replayed loop diverged from the recorded one")
        return el, len(traj), toks, h2d

    _, _, _, _, _, traj = run(False)   # warm-up pass (first launches, the pool's first touch, staging), recorded
    pa.padoc_check_device_errors(stream)
    e2e_s, steps, toks, h2d = run_replay(traj)
    pa.padoc_check_device_errors(stream)
    _, _, _, _, rec, _ = run(True)

    # algorithmic bytes of the loop: per step the decode minimum (each page's visible shared stream
    # once, private rows, Q in, O and LSE out) plus the append (the inputs' K and V rows written,
    # their queries read and laid out)
    nbytes = 0
    for host, stp in rec:
        info, S = stp.plan, int(stp.num_streams)
        sp = host[info.off_stream_page:info.off_stream_page + S]
        sh = host[info.off_shared_len:info.off_shared_len + S]
        pl = host[info.off_private_len:info.off_private_len + S]
        shared = int(np.maximum.reduceat(sh, np.r_[0, np.nonzero(np.diff(sp))[0] + 1]).sum())
        nbytes += (shared + int(pl.sum())) * Hkv * d * 4 + S * Hq * d * 4 + S * Hq * 4
        nbytes += S * Hkv * d * 4 + S * Hq * d * 4

    # (b) the recorded steps' ints in one device buffer (each step's words from a 256-byte boundary),
    # their launches (padoc_mpd_launch_step with the words already on the device: the append, then the
    # decode behind it) captured in a CUDA graph
    offs, n = [], 0
    for host, stp in rec:
        offs.append(n)
        n += (host.size + 63) // 64 * 64
    allh = np.zeros(max(n, 1), np.int32)
    for (host, stp), o in zip(rec, offs):
        allh[o:o + host.size] = host
    ints = torch.from_numpy(allh).to(dev)
    cmax = max(int(stp.num_streams) for _, stp in rec)
    ws_max = max(pa.padoc_decode_workspace_size(stp.plan) for _, stp in rec)
    ws = torch.empty(max(ws_max, 256), dtype=torch.uint8, device=dev)
    q_step = torch.empty((cmax, Hq, d), dtype=wl.dtype, device=dev)
    out = torch.empty((cmax, Hq, d), dtype=wl.dtype, device=dev)
    lse = torch.empty((cmax, Hq), dtype=torch.float32, device=dev)
    _, loop0 = admit_all()   # a fresh pool holding the prefixes, as at the loop's start
    torch.cuda.synchronize()
    views = [(stp, ints[o:o + int(stp.upload_words)]) for (host, stp), o in zip(rec, offs)]
    pool0 = pa.make_kv_pool(loop0.k_pool, loop0.v_pool)

    def replay(s):
        for stp, ints_d in views:
            pa.padoc_mpd_launch_step(stp, None, ints_d, pool0, kd, vd, qd, q_step, scale, out, lse, ws, s)

    replay(stream)
    pa.padoc_check_device_errors(stream)
    t0 = time.perf_counter()
    replay(stream)
    torch.cuda.synchronize()
    eager_s = time.perf_counter() - t0
    g = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream()
    with torch.cuda.graph(g, stream=cap):
        replay(torch.cuda.current_stream())
    g.replay()
    torch.cuda.synchronize()
    pa.padoc_check_device_errors(stream)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(physical_gpu_index(torch.cuda.current_device())) as clk:
        e0.record(stream)
        g.replay()
        e1.record(stream)
        torch.cuda.synchronize()
    pa.padoc_check_device_errors(stream)
    dev_s = e0.elapsed_time(e1) * 1e-3
    # per step: the append kernel, the decode grid and the merge
    launches = sum(1 + (1 if stp.plan.num_tc_items > 0 or stp.plan.num_warps > 0 else 0) + 1 for _, stp in rec)
    return dict(e2e_s=e2e_s, dev_s=dev_s, eager_s=eager_s, steps=steps, tokens=toks, bytes=nbytes, h2d=h2d,
                launches=launches, clocks=clk.summary(), pages=len(wl.pages), pool_blocks=nb)


# ------------------------------------------------------------------------------------------------
# Distributed plumbing (one process per GPU; no data-path collective: pages are independent)
# ------------------------------------------------------------------------------------------------

def physical_gpu_index(local: int) -> int:
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        ids = [x.strip() for x in vis.split(",") if x.strip()]
        if local < len(ids) and ids[local].isdigit():
            return int(ids[local])
    return local


def barrier(torch, world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(torch, world, x: float) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def cpu_baseline_decode(max_seconds=20.0):
    """The fp64 oracle as it stands on this host's cores, on a bounded sample of the serving batch:
    the first pages of the batch, as many as fit the time budget (at least one)."""
    import oracle
    from paper_2608_06146_gb300 import inputs
    wl_full = inputs.serving_batch(seed=3)
    scale = 1.0 / math.sqrt(wl_full.head_dim)
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    done_streams, elapsed, pages_used = 0, 0.0, 0
    for p in range(len(wl_full.pages)):
        wl = inputs.Workload("sample", [wl_full.pages[p]], 16, 2, 128, wl_full.dtype, "decode")
        di = inputs.decode_inputs(wl, 3)
        t0 = time.perf_counter()
        oracle.decode_pages(wl.pages, di, scale)
        elapsed += time.perf_counter() - t0
        done_streams += len(di.stream_page)
        pages_used += 1
        if elapsed > max_seconds / 2:
            break
    return {"value": done_streams / elapsed, "unit": "queries/s", "cores": cores, "kind": "oracle",
            "sample": f"decode step of the first {pages_used} of 32 serving-batch pages ({done_streams} branch "
                      f"queries x 16 heads), fp64, OpenMP, {elapsed:.2f} s"}


def decode_config(pages, streams, world):
    """The headline workload, as both arms name it."""
    return {"workload": "concurrent serving batch decode step: 32 pages, prefix U[1024,4096], Poisson(20) "
                        "branches/page, log-normal private KV (median 96, cap 2048)",
            "pages": pages, "streams_per_gpu": streams, "num_q_heads": 16, "num_kv_heads": 2, "head_dim": 128,
            "block_size": 16, "parallelism": f"replicas x{world} (pages per GPU)",
            "l2": "inputs rotate over replicas in distinct memory totalling more than 4x L2"}


def run_reference(args):
    """The oracle as the reference arm: each step is the decode step of the whole 32-page serving
    batch (the headline's workload), fp64 on the host cores."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import oracle
    from paper_2608_06146_gb300 import inputs
    oracle.build()
    wl = inputs.serving_batch(seed=3)
    di = inputs.decode_inputs(wl, 3, pool_slack=1.0)
    scale = 1.0 / math.sqrt(wl.head_dim)
    S = len(di.stream_page)

    def step():
        oracle.decode_pages(wl.pages, di, scale)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = (time.perf_counter() - t0) / args.steps
    value = S / dt
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "queries/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": decode_config(len(wl.pages), S, args.gpus),
            "cpu_baseline": {"value": value, "unit": "queries/s", "cores": cores, "kind": "oracle",
                             "sample": f"the whole 32-page serving batch, {S} branch queries x 16 heads per step"},
            "e2e": {"value": value, "unit": "queries/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="padoc", choices=["padoc", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--only", default="all", choices=["all", "decode", "prefill", "prefill_bwd", "loop",
                                                      "chunk_prefill", "variants", "decode_e4m3", "replicas"])
    ap.add_argument("--replicas", type=int, default=0, help="decode input replicas (0: enough to exceed 4x L2)")
    ap.add_argument("--shape", choices=["decode_page", "dense_page"], default=None,
                    help="with --only replicas: that page shape alone")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-steady", action="store_true", help="skip the long back-to-back decode run")
    ap.add_argument("--tc-ctas", type=int, default=0, help="tensor-core decode CTAs (0: one per SM)")
    ap.add_argument("--warp-ctas", type=int, default=0, help="warp-kernel decode CTAs (0: one per SM)")
    ap.add_argument("--split-tokens", type=int, default=0, help="decode shared-stream split (0: library default)")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)

    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
    torch.cuda.set_device(local)
    dev = f"cuda:{local}"

    # CPU baseline first: the oracle runs on the host cores before any GPU work of this process
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        cpu = cpu_baseline_decode()

    from paper_2608_06146_gb300 import build as pbuild
    pbuild.build()
    if args.only == "variants":   # the two extra report lines alone
        a = bench_decode(args, torch, dev, rank, world, layout_streams=True)
        b = bench_prefill(args, torch, dev, rank, world, shuffle=True)
        if rank == 0:
            print(json.dumps({"decode_with_layout_streams_us": a["ms"] * 1e3, "streams": a["streams"],
                              "prefill_shuffled_ms": b["ms"], "prefill_shuffled_tflops": b["flops"] / (b["ms"] * 1e-3) / 1e12}))
        return 0
    if args.only == "replicas":
        for shape in (args.shape,) if args.shape else ("decode_page", "dense_page"):
            r = bench_decode_replicas(args, torch, dev, rank, world, shape)
            if rank == 0:
                print(json.dumps({"shape": shape, "pages": r["pages"], "streams": r["streams"], "us": r["ms"] * 1e3,
                                  "queries_per_s": r["streams"] / (r["ms"] * 1e-3),
                                  "hbm_frac": r["bytes"] / (r["ms"] * 1e-3) / 1e9 / load_peaks()[0]["hbm_gbs"],
                                  "tc_items": r["tc_items"], "warp_items": r["warp_items"]}))
        return 0
    if args.only == "decode_e4m3":
        e = bench_decode_e4m3(args, torch, dev, rank, world)
        if rank == 0:
            print(json.dumps({"decode_e4m3_us": e["ms"] * 1e3, "queries_per_s": e["streams"] / (e["ms"] * 1e-3),
                              "hbm_gbs": e["bytes"] / (e["ms"] * 1e-3) / 1e9, "bytes": e["bytes"]}))
        return 0
    if args.only == "loop":
        lp = bench_loop(args, torch, dev, rank, world)
        if rank == 0:
            print(json.dumps({"loop_tokens_per_s_e2e": lp["tokens"] / lp["e2e_s"],
                              "loop_tokens_per_s_device": lp["tokens"] / lp["dev_s"], **{k: lp[k] for k in
                              ("steps", "tokens", "e2e_s", "dev_s", "eager_s", "bytes", "h2d", "launches")}}))
        return 0
    if args.only in ("prefill", "prefill_bwd", "chunk_prefill"):
        fn = {"prefill": bench_prefill, "prefill_bwd": bench_prefill_bwd,
              "chunk_prefill": bench_chunk_prefill}[args.only]
        p = fn(args, torch, dev, rank, world)
        pms = max_over_ranks(torch, world, p["ms"])
        if rank == 0:
            print(json.dumps({f"{args.only}_ms": pms, "tflops": p["flops"] * world / (pms * 1e-3) / 1e12}))
        return 0
    d = bench_decode(args, torch, dev, rank, world)
    p = None if args.only == "decode" else bench_prefill(args, torch, dev, rank, world)
    pb = None if args.only == "decode" else bench_prefill_bwd(args, torch, dev, rank, world)
    def variant(fn, **kw):   # an extra report line: a failure is recorded, the headline stands
        try:
            return fn(args, torch, dev, rank, world, **kw)
        except Exception as e:  # noqa: BLE001
            return {"error": f"{type(e).__name__}: {e}"[:300]}

    dl = None if args.only == "decode" else variant(bench_decode, layout_streams=True)
    d8 = None if args.only == "decode" else variant(bench_decode_e4m3)
    reps = {} if args.only == "decode" else {k: variant(bench_decode_replicas, shape=k)
                                               for k in ("decode_page", "dense_page")}
    ps = None if args.only == "decode" else variant(bench_prefill, shuffle=True)
    cp = None if args.only == "decode" else variant(bench_chunk_prefill)
    lp = None if args.only == "decode" else variant(bench_loop)

    peaks, peak_src = load_peaks()
    ms = max_over_ranks(torch, world, d["ms"])
    e2e_ms = max_over_ranks(torch, world, d["e2e_ms"] if d["e2e_ms"] is not None else float("nan"))
    total_streams = d["streams"] * world   # each rank decodes its own batch of the same shape
    value = total_streams / (ms * 1e-3)
    achieved = d["bytes"] / (d["ms"] * 1e-3) / 1e9
    roof = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": achieved / peaks["hbm_gbs"], "traffic": TRAFFIC_BYTES["decode"],
            "peak_source": f"{peak_src} hbm_gbs", "kernel": "decode step (tensor-core shared-stream kernel + warp kernel + split-K merge)",
            "algorithmic_bytes": d["bytes"], "frac_of_nominal_8tbs": achieved / 8000.0}
    line = {"metric": METRIC, "value": value, "unit": "queries/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": decode_config(d["pages"], d["streams"], world),
            "l2_replicas": d["replicas"],
            "timing": "the K steps replayed from CUDA graphs (steps as programmatic dependents of one another, as "
                      "when launched one by one) between one pair of CUDA events, right after the long run "
                      "(decode_steady) with no idle gap",
            "roofline": roof, "gpu_launches": d["launches"] * args.steps, "clocks": d["clocks"],
            "e2e": {"value": total_streams / (e2e_ms * 1e-3), "unit": "queries/s", "h2d_bytes_per_step": d["h2d"],
                    "d2h_bytes_per_step": d["d2h"]}}
    if d.get("steady"):
        sd = d["steady"]
        sach = d["bytes"] / (sd["median_ms"] * 1e-3) / 1e9
        line["decode_steady"] = {
            "value": total_streams / (max_over_ranks(torch, world, sd["median_ms"]) * 1e-3), "unit": "queries/s",
            "median_ms_per_step": sd["median_ms"], "min_ms_per_step": sd["min_ms"], "max_ms_per_step": sd["max_ms"],
            "mean_ms_per_step": sd["mean_ms"], "steps": sd["steps"],
            "how": f"{sd['replays']} replays of a CUDA graph of {sd['graph_steps']} back-to-back decode steps over the "
                   "same rotating replicas, each replay between its own CUDA events; per-step median over replays",
            "roofline": {"bound": "hbm", "achieved": sach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": sach / peaks["hbm_gbs"], "algorithmic_bytes": d["bytes"]}}
    if cpu is not None:
        line["cpu_baseline"] = cpu
    if p is not None:
        pms = max_over_ranks(torch, world, p["ms"])
        tflops = p["flops"] * world / (pms * 1e-3) / 1e12
        line["prefill"] = {"value": tflops, "unit": "TFLOP/s", "ms_per_step": pms, "steps": p["steps"],
                           "workload": "packed ancestor prefill, 8 pages x 4096 tokens (32768), unmasked-entry FLOPs",
                           "l2": "flushed between steps",
                           "roofline": {"bound": "tensor", "achieved": p["flops"] / (p["ms"] * 1e-3) / 1e12,
                                        "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                                        "frac": p["flops"] / (p["ms"] * 1e-3) / 1e12 / peaks["bf16_tflops"],
                                        "traffic": TRAFFIC_BYTES["prefill"],
                                        "peak_source": f"{peak_src} bf16_tflops (burst)",
                                        "algorithmic_flops": p["flops"]}}
    if pb is not None:
        bms = max_over_ranks(torch, world, pb["ms"])
        achieved = pb["flops"] / (pb["ms"] * 1e-3) / 1e12
        line["prefill_bwd"] = {"value": pb["flops"] * world / (bms * 1e-3) / 1e12, "unit": "TFLOP/s", "ms_per_step": bms,
                               "steps": pb["steps"],
                               "workload": "gradients (dQ, dK, dV) of the packed ancestor prefill, 8 pages x 4096 "
                                           "tokens, 2.5x the forward's unmasked-entry FLOPs",
                               "l2": "flushed between steps",
                               "roofline": {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops"],
                                            "unit": "TFLOP/s", "frac": achieved / peaks["bf16_tflops"],
                                            "traffic": TRAFFIC_BYTES["prefill_bwd"],
                                            "peak_source": f"{peak_src} bf16_tflops (burst)",
                                            "algorithmic_flops": pb["flops"]}}
    if dl is not None:
        if "error" in dl:
            line["decode_with_layout_streams"] = dl
        else:
            dms = max_over_ranks(torch, world, dl["ms"])
            ach = dl["bytes"] / (dl["ms"] * 1e-3) / 1e9
            line["decode_with_layout_streams"] = {
                "value": dl["streams"] * world / (dms * 1e-3), "unit": "queries/s", "ms_per_step": dms,
                "streams_per_gpu": dl["streams"],
                "workload": "the serving-batch decode step with every page's layout stream decoded too "
                            "(branches + layout streams; the headline counts branches only)",
                "roofline": {"bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                             "frac": ach / peaks["hbm_gbs"], "traffic": None, "algorithmic_bytes": dl["bytes"]}}
    for shape, key, desc in (("decode_page", "decode_one_page_replicas",
                              "one-page decode shape (P = 2048 = 1792 visual + 256 prompt, layout stream 256, 16 "
                              "branches, private KV U[16,256])"),
                             ("dense_page", "decode_dense_page_replicas",
                              "dense-page decode shape (P = 4096, layout stream 512, 64 branches, log-normal private "
                              "KV, median 64, cap 1024)")):
        r = reps.get(shape)
        if r is None:
            continue
        if "error" in r:
            line[key] = r
            continue
        rms = max_over_ranks(torch, world, r["ms"])
        ach = r["bytes"] / (r["ms"] * 1e-3) / 1e9
        line[key] = {"value": r["streams"] * world / (rms * 1e-3), "unit": "queries/s", "ms_per_step": rms,
                     "pages": r["pages"], "streams_per_gpu": r["streams"], "clocks": r["clocks"],
                     "tc_items": r["tc_items"], "warp_items": r["warp_items"],
                     "workload": f"{r['pages']} replicas of the {desc}, each with its own K/V/Q in distinct memory, "
                                 "decoded as one batch per step (the batch's cache > 4x L2)",
                     "roofline": {"bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                                  "frac": ach / peaks["hbm_gbs"], "traffic": None, "algorithmic_bytes": r["bytes"]}}
    if d8 is not None and "error" in d8:
        line["decode_e4m3"] = d8
    elif d8 is not None:
        ems = max_over_ranks(torch, world, d8["ms"])
        ach = d8["bytes"] / (d8["ms"] * 1e-3) / 1e9
        line["decode_e4m3"] = {
            "value": d8["streams"] * world / (ems * 1e-3), "unit": "queries/s", "ms_per_step": ems,
            "streams_per_gpu": d8["streams"], "replicas": d8["replicas"], "clocks": d8["clocks"],
            "workload": "the serving-batch decode step over the FP8 (E4M3) KV cache (codes + one fp32 scale per "
                        "(block, KV head)), quantized from the same bf16 cache",
            "roofline": {"bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": ach / peaks["hbm_gbs"], "traffic": TRAFFIC_BYTES["decode_e4m3"],
                         "algorithmic_bytes": d8["bytes"],
                         "bytes_rule": "each page's visible shared stream once and every private row once at 1 byte "
                                       "per K/V element, plus a 4-byte K and V scale per (16-token block, KV head), Q "
                                       "in, O and LSE out"}}
    if ps is not None and p is not None:
        if "error" in ps:
            line["prefill"]["shuffled_branches"] = ps
        else:
            sms = max_over_ranks(torch, world, ps["ms"])
            line["prefill"]["shuffled_branches"] = {
                "value": ps["flops"] * world / (sms * 1e-3) / 1e12, "unit": "TFLOP/s", "ms_per_step": sms,
                "workload": "the same packed prefill with each page's branches permuted (fork offsets not "
                            "monotone in the branch index)",
                "frac": ps["flops"] / (ps["ms"] * 1e-3) / 1e12 / peaks["bf16_tflops"]}
    if cp is not None and "error" in cp:
        line["branch_prefill"] = cp
    elif cp is not None:
        cms = max_over_ranks(torch, world, cp["ms"])
        achieved = cp["flops"] / (cp["ms"] * 1e-3) / 1e12
        line["branch_prefill"] = {
            "value": cp["flops"] * world / (cms * 1e-3) / 1e12, "unit": "TFLOP/s", "ms_per_step": cms,
            "tokens_per_s": cp["tokens"] * world / (cms * 1e-3), "steps": cp["steps"],
            "workload": "branch prefill over the paged cache of the 32 serving-batch pages: every branch's tokens as "
                        "one chunk from its branch-initialization token, every layout stream as one shared-stream "
                        f"chunk ({cp['chunks']} chunks, {cp['tokens']} query tokens), unmasked-entry FLOPs",
            "l2": "flushed between steps",
            "roofline": {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                         "frac": achieved / peaks["bf16_tflops"], "traffic": None,
                         "peak_source": f"{peak_src} bf16_tflops (burst)", "algorithmic_flops": cp["flops"]}}
    if lp is not None and "error" in lp:
        line["loop"] = lp
    elif lp is not None:
        tokens = lp["tokens"] * world
        e2e_s = max_over_ranks(torch, world, lp["e2e_s"])
        dev_s = max_over_ranks(torch, world, lp["dev_s"])
        achieved = lp["bytes"] / lp["dev_s"] / 1e9
        line["loop"] = {"value": tokens / e2e_s, "unit": "decoded tokens/s", "seconds": e2e_s, "steps": lp["steps"],
                        "tokens_per_gpu": lp["tokens"],
                        "workload": "Algorithm 1 over the 32 serving-batch pages: every layout stream and branch "
                                    "decoded from its first input to its EOS (prefixes admitted untimed)",
                        "h2d_bytes_per_step": lp["h2d"] / lp["steps"], "d2h_bytes_per_step": 0,
                        "device": {"value": tokens / dev_s, "unit": "decoded tokens/s", "seconds": dev_s,
                                   "gpu_launches": lp["launches"], "clocks": lp["clocks"],
                                   "eager_replay_s": lp["eager_s"],
                                   "how": "the same steps' append + decode launches, captured once in a CUDA graph "
                                          "from per-step inputs already on the device, replayed"},
                        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                                     "frac": achieved / peaks["hbm_gbs"], "traffic": None,
                                     "peak_source": f"{peak_src} hbm_gbs", "algorithmic_bytes": lp["bytes"]}}
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
