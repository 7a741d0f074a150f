// prefill_bwd_tc.cu -- gradients of the packed ancestor prefill on the 5th-generation tensor cores
// (App. C.1: the backward of the tree-varlen attention; Sec. 3.2 visibility), in two passes that
// need neither a gather nor atomics.
//
// With c = scale * log2(e), lse2 = lse * log2(e) and D = rowsum(dO * O) per query row and head
// (-lse2 and D precomputed per head, [Hq][t_pad], padded rows -lse2 = -inf so that their P is 0):
//   P = exp2(S c - lse2),  dS = P (dP - D),  S = Q K^T,  dP = dO V^T.
//
// dK/dV pass: one CTA per (128-key k-tile, KV head), k-tiles taken in the key-major map's order
//   (most work first); a unit with more than PADOC_BWD_SPLIT_STEPS steps runs as two CTAs over its
//   two halves of steps, which write fp32 partials that prefill_bwd_dkv_merge_kernel adds (the
//   heaviest units otherwise set the pass's tail). K and V of the tile sit in tensor memory as A
//   operands for the whole walk.
//   For every (32-row q-tile that sees the k-tile, query head reading the KV head) step the tensor
//   cores form S^T = K Q^T and dP^T = V dO^T (M = 128 keys, N = 32 queries, B from shared memory),
//   the softmax warps write P^T and dS^T back into tensor memory as bf16, and dV += P^T dO,
//   dK += dS^T Q accumulate in tensor memory over the whole walk. Every query that sees a
//   shared-stream key (the stream's later tokens and each branch forked after it) therefore adds
//   into that key's gradient inside one CTA: the scatter-add of the gather's backward, with nothing
//   scattered.
// dQ pass: one CTA per (128-row q-tile, query head), heavier q-tiles first, Q and dO resident in
//   tensor memory. It walks the query-major map of 32-key k-tiles: S = Q K^T, dP = dO V^T, dS written
//   back as bf16, dQ += dS K.
//
// Every MMA reads at most one operand from shared memory (the other lives in tensor memory), which
// keeps the narrow steps at the tensor cores' rate instead of shared memory's. Tensor memory holds
// the resident A operands (128 columns), the accumulators (dV and dK: 256; dQ: 128) and, in what
// is left, as many step buffers (S and dP, 2 x 32 columns each) as fit: 2 in the dK/dV pass, 4 in
// the dQ pass. While the softmax warps turn step u into P and dS, the tensor cores run the
// accumulating MMAs of step u-1 and the S and dP of the steps after u. A softmax warp owns 32 TMEM
// lanes (rows) and one 16-column half of a step and packs its 16 bf16 results into the first 8
// columns of its own half, so no warp overwrites a column another warp still has to read; the
// accumulating MMAs read the two k-slices at columns 0 and 16 of the buffer.
//
// Warp roles (320 threads): warps 0-7 softmax and epilogue (they also store the resident operands
// into tensor memory), warp 8 TMA producer, warp 9 TMEM allocation and MMA issue (converged warp,
// one elected lane issues). Every wait is bounded; a wait that runs out records an error and all
// roles leave their loops, the MMA warp waits for its MMAs, the producer for its copies, and tensor
// memory is released.
#include <math.h>

#include <algorithm>
#include <type_traits>

#include "common.cuh"
#include "tc.cuh"

namespace {

constexpr int kD = 128;
constexpr int kThreads = 320;
constexpr uint32_t kTmemCols = 512;

struct BwdParams {
    const int32_t *spans, *ptr, *idx, *order;
    const int8_t *kind;
    float *lt, *dt;                     // [Hq][t_pad]: -lse2 and D (written by the dQ pass, read by the dK/dV pass)
    const __nv_bfloat16 *o;             // the forward's output (dQ pass: D = dO . O)
    const float *lse;                   // the forward's log-sum-exp, natural log, [T][Hq]
    const __nv_bfloat16 *a0, *a1;       // the pass's tensor-memory operands: dQ pass Q, dO; dK/dV pass K, V
    int64_t T, t_pad;
    int32_t num_q_heads, num_kv_heads, num_tiles;
    float scale_log2, scale;
    __nv_bfloat16 *out0, *out1;         // dK/dV pass: dK, dV; dQ pass: dQ
    float *split;                       // dK/dV pass: fp32 partials of the split units
    int32_t split_units;                // dK/dV pass: units of the key-major order below this may split
    int *err;
};

__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, int *err, int site, volatile int *abort_flag)
{
    if (*abort_flag) return false;
    if (mbar_wait_bounded(bar, parity, err, site)) return true;
    *abort_flag = 1;
    return false;
}

// TMEM column of k-slice k (16 values) of a W-wide bf16 operand written by the softmax warps: column
// half c packs its W/2 values into the first W/4 columns of its own half.
template <int W>
__device__ __forceinline__ uint32_t slice_col(int k)
{
    constexpr int per_half = W / 32;
    return (uint32_t)((k / per_half) * (W / 2) + (k % per_half) * 8);
}

template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t (&r)[N])
{
    static_assert(N == 16 || N == 32, "16 or 32 columns");
    if constexpr (N == 32) tmem_ld32(taddr, r); else tmem_ld16(taddr, r);
}
template <int N>
__device__ __forceinline__ void tmem_st_cols(uint32_t taddr, const uint32_t (&r)[N])
{
    static_assert(N == 8 || N == 16, "8 or 16 columns");
    if constexpr (N == 16) tmem_st16(taddr, r); else tmem_st8(taddr, r);
}

__device__ __forceinline__ void store_row_bf16(__nv_bfloat16 *dst, const uint32_t (&o)[32], float mul)
{
#pragma unroll
    for (int i = 0; i < 32; i += 8) {
        uint4 w;
        w.x = pack_bf16x2(__uint_as_float(o[i]) * mul, __uint_as_float(o[i + 1]) * mul);
        w.y = pack_bf16x2(__uint_as_float(o[i + 2]) * mul, __uint_as_float(o[i + 3]) * mul);
        w.z = pack_bf16x2(__uint_as_float(o[i + 4]) * mul, __uint_as_float(o[i + 5]) * mul);
        w.w = pack_bf16x2(__uint_as_float(o[i + 6]) * mul, __uint_as_float(o[i + 7]) * mul);
        *reinterpret_cast<uint4 *>(dst + i) = w;
    }
}

// Stores 64 bf16 of a row (global, 16-byte aligned; zeros when src is null) into 32 TMEM columns of
// the calling thread's lane: the K-major A-operand layout (column c holds elements 2c, 2c+1).
__device__ __forceinline__ void row_to_tmem(uint32_t taddr, const __nv_bfloat16 *src)
{
    uint32_t w[32];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const uint4 x = src ? reinterpret_cast<const uint4 *>(src)[i] : make_uint4(0u, 0u, 0u, 0u);
        w[4 * i] = x.x; w[4 * i + 1] = x.y; w[4 * i + 2] = x.z; w[4 * i + 3] = x.w;
    }
    tmem_st32(taddr, w);
}

__device__ __forceinline__ int clamp_w(int x, int w) { return min(max(x, 0), w); }

// 32 x 32 bit-matrix transpose across a warp: lane r holds row r (bit c = element (r, c)); on return
// lane r holds column r (bit c = element (c, r)). Five exchange rounds, each swapping the off-diagonal
// j x j blocks between lanes r and r ^ j.
__device__ __forceinline__ uint32_t transpose32_warp(uint32_t x, int lane)
{
    uint32_t m = 0x0000FFFFu;
#pragma unroll
    for (int j = 16; j != 0; j >>= 1) {
        const uint32_t o = __shfl_xor_sync(0xffffffffu, x, j);
        if (lane & j) x ^= ((o >> j) ^ x) & m;
        else x ^= (((x >> j) ^ o) & m) << j;
        m ^= m << (j >> 1);
    }
    return x;
}

// ================================================================================================
// dK/dV pass
// ================================================================================================
namespace dkv {
constexpr int kKT = PADOC_BWD_DKV_K_TILE;   // 128 keys: the M of every MMA
constexpr int kQT = PADOC_BWD_DKV_Q_TILE;   // 64 queries per step
constexpr int kStages = 3;
constexpr uint32_t kColS = 0, kColDP = 128, kColAcc0 = 256, kColAcc1 = 384;
constexpr int kKPanel = kKT * 128;           // [128 rows][64 bf16]
constexpr int kQPanel = kQT * 128;           // [64 rows][64 bf16]
constexpr int kKTile = 2 * kKPanel;
constexpr int kQTile = 2 * kQPanel;
constexpr int kAuxBytes = 2 * kQT * 4 + kQT * 16;   // lse2[64], D[64], spans[64][4]
enum {
    B_KV = 0,
    B_QFULL = 1,                  // [stage]
    B_QEMPTY = 1 + kStages,       // [stage]
    B_SFULL = 1 + 2 * kStages,    // [step parity]
    B_PFULL = 3 + 2 * kStages,    // [step parity], 256 arrivals
    B_FINAL = 5 + 2 * kStages,
    B_COUNT = 6 + 2 * kStages
};
constexpr size_t kSmemBytes = 1024 + 2 * (size_t)kKTile + 2 * (size_t)kStages * kQTile + (size_t)kStages * kAuxBytes +
                              B_COUNT * 8 + 64;
}  // namespace dkv

__global__ void __launch_bounds__(kThreads, 1)
prefill_bwd_dkv_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap gmap,
                       const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                       const BwdParams prm)
{
    using namespace dkv;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *sk = smem;
    uint8_t *sv = sk + kKTile;
    uint8_t *sq = sv + kKTile;                 // [stage] Q step tiles
    uint8_t *sg = sq + kStages * kQTile;       // [stage] dO step tiles
    uint8_t *aux = sg + kStages * kQTile;      // [stage] lse2, D, spans
    uint64_t *bars = (uint64_t *)(aux + kStages * kAuxBytes);
    uint32_t *tmem_slot = (uint32_t *)(bars + B_COUNT);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int hkv = prm.num_kv_heads, group = prm.num_q_heads / hkv;
    // CTA b: KV head b % hkv of the (b / hkv) % 2-th half of unit b / (2 hkv) of the key-major order;
    // a unit of more than PADOC_BWD_SPLIT_STEPS steps (among the first split_units) runs as two
    // halves that write fp32 partials, the others as one CTA (the second CTA leaves at once)
    const int unit = (int)(blockIdx.x / (2 * hkv)), half = (int)((blockIdx.x / hkv) & 1), g = (int)(blockIdx.x % hkv);
    const int kt = prm.order[unit];
    const int e0 = prm.ptr[kt], ne = prm.ptr[kt + 1] - e0;
    const bool split = ne * group > PADOC_BWD_SPLIT_STEPS && unit < prm.split_units;
    if (half == 1 && !split) return;
    const int ub = half ? ne * group / 2 : 0;                               // first step of this CTA
    const int nu = split ? (half ? ne * group - ub : ne * group / 2) : ne * group;
    auto bar = [&](int i) { return smem_u32(&bars[i]); };

    if (tid == 0) {
        for (int i = 0; i < B_COUNT; ++i) mbar_init(bar(i), (i == B_PFULL || i == B_PFULL + 1) ? 256 : 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 9) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 8) {
        // ---------------------------------------------------------------- TMA producer
        if (lane == 0 && nu > 0) {
            tma_prefetch_desc(&qmap);
            tma_prefetch_desc(&gmap);
            tma_prefetch_desc(&kmap);
            tma_prefetch_desc(&vmap);
            mbar_arrive_expect_tx(bar(B_KV), 2 * kKTile);
            tma_load_2d(smem_u32(sk), &kmap, g * kD, kt * kKT, bar(B_KV));
            tma_load_2d(smem_u32(sk) + kKPanel, &kmap, g * kD + 64, kt * kKT, bar(B_KV));
            tma_load_2d(smem_u32(sv), &vmap, g * kD, kt * kKT, bar(B_KV));
            tma_load_2d(smem_u32(sv) + kKPanel, &vmap, g * kD + 64, kt * kKT, bar(B_KV));
            int issued = 0;
            for (int u = 0; u < nu; ++u) {
                const int s = u % kStages;
                if (u >= kStages && !wait_or_abort(bar(B_QEMPTY + s), (u / kStages - 1) & 1, prm.err, 50, abort_flag))
                    break;
                const int e = e0 + (ub + u) / group, h = g * group + (ub + u) % group;
                const int q0 = prm.idx[e] * kQT;
                const int nsp = prm.kind[e] == PADOC_TILE_FULL ? 0 : min(kQT, (int)(prm.T - q0)) * 16;
                const uint32_t fb = bar(B_QFULL + s);
                const uint32_t qb = smem_u32(sq + s * kQTile), gb = smem_u32(sg + s * kQTile);
                const uint32_t ab = smem_u32(aux + s * kAuxBytes);
                mbar_arrive_expect_tx(fb, 2 * kQTile + 2 * kQT * 4 + nsp);
                tma_load_2d(qb, &qmap, h * kD, q0, fb);
                tma_load_2d(qb + kQPanel, &qmap, h * kD + 64, q0, fb);
                tma_load_2d(gb, &gmap, h * kD, q0, fb);
                tma_load_2d(gb + kQPanel, &gmap, h * kD + 64, q0, fb);
                bulk_load(ab, prm.lt + (size_t)h * prm.t_pad + q0, kQT * 4, fb);
                bulk_load(ab + kQT * 4, prm.dt + (size_t)h * prm.t_pad + q0, kQT * 4, fb);
                if (nsp) bulk_load(ab + 2 * kQT * 4, prm.spans + 4 * (size_t)q0, (uint32_t)nsp, fb);
                issued = u + 1;
            }
            // copies still in flight must land before the CTA's shared memory is released
            mbar_wait_bounded(bar(B_KV), 0, prm.err, 51);
            for (int u = (issued > kStages ? issued - kStages : 0); u < issued; ++u)
                mbar_wait_bounded(bar(B_QFULL + u % kStages), (u / kStages) & 1, prm.err, 52);
        }
    } else if (warp == 9) {
        // ---------------------------------------------------------------- MMA issuer (whole warp)
        if (nu > 0) {
            constexpr uint32_t idS = umma_idesc_bf16(128, kQT, false);
            constexpr uint32_t idAcc = umma_idesc_bf16(128, kD, true);
            const uint64_t dK = umma_desc_sw128(smem_u32(sk), 16, 1024);
            const uint64_t dV = umma_desc_sw128(smem_u32(sv), 16, 1024);
            auto wait_w = [&](int b, uint32_t parity, int site) {
                const bool r = wait_or_abort(bar(b), parity, prm.err, site, abort_flag);
                return __all_sync(0xffffffffu, r);
            };
            // S^T and dP^T of step u into the parity-(u & 1) columns
            auto issue_s = [&](int u) {
                const int s = u % kStages;
                const uint32_t b = (uint32_t)(u & 1) * 64;
                const uint64_t dq = umma_desc_sw128(smem_u32(sq + s * kQTile), 16, 1024);
                const uint64_t dg = umma_desc_sw128(smem_u32(sg + s * kQTile), 16, 1024);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {
                    const uint32_t oa = ((ks >> 2) * kKPanel + (ks & 3) * 32) >> 4;
                    const uint32_t ob = ((ks >> 2) * kQPanel + (ks & 3) * 32) >> 4;
                    umma_bf16_ss_warp(tmem + kColS + b, dK + oa, dq + ob, idS, ks > 0);
                }
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {
                    const uint32_t oa = ((ks >> 2) * kKPanel + (ks & 3) * 32) >> 4;
                    const uint32_t ob = ((ks >> 2) * kQPanel + (ks & 3) * 32) >> 4;
                    umma_bf16_ss_warp(tmem + kColDP + b, dV + oa, dg + ob, idS, ks > 0);
                }
                umma_commit_warp(bar(B_SFULL + (u & 1)));
            };
            bool ok = wait_w(B_KV, 0, 60);
            for (int u = 0; ok && u < 2 && u < nu; ++u) {
                ok = wait_w(B_QFULL + u % kStages, (u / kStages) & 1, 61);
                if (ok) {
                    tc_fence_after();
                    issue_s(u);
                }
            }
            for (int u = 0; ok && u < nu; ++u) {
                const int s = u % kStages;
                const uint32_t b = (uint32_t)(u & 1) * 64;
                if (!wait_w(B_PFULL + (u & 1), (u >> 1) & 1, 62)) { ok = false; break; }
                tc_fence_after();
                // the step's Q and dO as MN-major B operands (N = head dim, K = the 64 queries)
                const uint64_t gmn = umma_desc_sw128(smem_u32(sg + s * kQTile), kQPanel, 1024);
                const uint64_t qmn = umma_desc_sw128(smem_u32(sq + s * kQTile), kQPanel, 1024);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    umma_bf16_ts_warp(tmem + kColAcc0, tmem + kColS + b + slice_col<kQT>(kk), gmn + kk * (2048 >> 4), idAcc,
                                      (u > 0 || kk > 0));
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    umma_bf16_ts_warp(tmem + kColAcc1, tmem + kColDP + b + slice_col<kQT>(kk), qmn + kk * (2048 >> 4), idAcc,
                                      (u > 0 || kk > 0));
                umma_commit_warp(bar(B_QEMPTY + s));
                if (u + 2 < nu) {
                    if (!wait_w(B_QFULL + (u + 2) % kStages, ((u + 2) / kStages) & 1, 63)) { ok = false; break; }
                    tc_fence_after();
                    issue_s(u + 2);
                }
            }
            // every MMA issued above must complete before tensor memory is read or released
            umma_commit_warp(bar(B_FINAL));
            mbar_wait_bounded(bar(B_FINAL), 0, prm.err, 64);
        }
    } else {
        // ---------------------------------------------------------------- softmax + epilogue
        const int lq = warp & 3, ch = warp >> 2;          // TMEM lane quarter, column half
        const int key = kt * kKT + lq * 32 + lane;
        const uint32_t lanes = (uint32_t)(lq * 32) << 16;
        const float c = prm.scale_log2;
        auto wait_all = [&](int b, uint32_t parity, int site) {
            const bool r = wait_or_abort(bar(b), parity, prm.err, site, abort_flag);
            return __all_sync(0xffffffffu, r);
        };
        bool ok = true;
        for (int u = 0; u < nu; ++u) {
            const int s = u % kStages;
            const uint32_t b = (uint32_t)(u & 1) * 64 + 32 * ch;
            const int e = e0 + (ub + u) / group;
            const bool partial = prm.kind[e] != PADOC_TILE_FULL;
            const int qbase = prm.idx[e] * kQT + 32 * ch;
            if (!wait_all(B_SFULL + (u & 1), (u >> 1) & 1, 70) || !wait_all(B_QFULL + s, (u / kStages) & 1, 71)) {
                ok = false;
                break;
            }
            tc_fence_after();
            uint32_t sr[32], dr[32];
            tmem_ld32(tmem + lanes + kColS + b, sr);
            tmem_ld32(tmem + lanes + kColDP + b, dr);
            const float4 *la = reinterpret_cast<const float4 *>(aux + s * kAuxBytes) + 8 * ch;
            const float4 *da = reinterpret_cast<const float4 *>(aux + s * kAuxBytes + kQT * 4) + 8 * ch;
            const int4 *sp = reinterpret_cast<const int4 *>(aux + s * kAuxBytes + 2 * kQT * 4) + 32 * ch;
            uint32_t vis = 0xffffffffu;
            if (partial) {   // (warp-uniform)
                // lane i: which of the warp's 32 keys query qbase + i sees (its two spans as bit
                // intervals); a 32 x 32 bit transpose across the warp then gives each key's bits over
                // the 32 queries
                const int64_t rem = prm.T - qbase;   // query columns past T hold no spans
                const int nvalid = rem <= 0 ? 0 : (rem >= 32 ? 32 : (int)rem);
                const int kbase = kt * kKT + lq * 32;
                uint32_t x = 0u;
                if (lane < nvalid) {
                    const int4 w = sp[lane];
                    const int lo0 = clamp_w(w.x - kbase, 32), lo1 = clamp_w(w.z - kbase, 32);
                    x = interval_bits(lo0, max(clamp_w(w.y - kbase, 32) - lo0, 0), 0) |
                        interval_bits(lo1, max(clamp_w(w.w - kbase, 32) - lo1, 0), 0);
                }
                vis = transpose32_warp(x, lane);
            }
            tmem_ld_wait();
            uint32_t pk[16], dk[16];
            const uint64_t c2 = f2_pack(c, c);
            // two query columns per packed instruction: P = exp2(S c - lse2), dS = P (dP - D)
            auto column_pairs = [&](auto masked) {
#pragma unroll
                for (int i4 = 0; i4 < 8; ++i4) {
                    const float4 l4 = la[i4], d4 = da[i4];
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
                        const int i = 4 * i4 + 2 * j;
                        float x0, x1;
                        f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[i]), __uint_as_float(sr[i + 1])), c2,
                                         j ? f2_pack(l4.z, l4.w) : f2_pack(l4.x, l4.y)), x0, x1);
                        float p0 = fast_exp2(x0), p1 = fast_exp2(x1);
                        if (decltype(masked)::value) {
                            p0 = (vis >> i) & 1u ? p0 : 0.f;
                            p1 = (vis >> (i + 1)) & 1u ? p1 : 0.f;
                        }
                        const uint64_t t = f2_sub(f2_pack(__uint_as_float(dr[i]), __uint_as_float(dr[i + 1])),
                                                  j ? f2_pack(d4.z, d4.w) : f2_pack(d4.x, d4.y));
                        float d0, d1;
                        f2_unpack(f2_mul(f2_pack(p0, p1), t), d0, d1);
                        pk[i >> 1] = pack_bf16x2(p0, p1);
                        dk[i >> 1] = pack_bf16x2(d0, d1);
                    }
                }
            };
            if (partial) column_pairs(std::true_type{}); else column_pairs(std::false_type{});
            tmem_st16(tmem + lanes + kColS + b, pk);
            tmem_st16(tmem + lanes + kColDP + b, dk);
            tmem_st_wait();
            tc_fence_before();
            mbar_arrive(bar(B_PFULL + (u & 1)));
        }
        // epilogue: column half 0 writes dV, half 1 writes dK (times scale), one key row per thread;
        // a split unit's halves write their fp32 sums instead ([unit][g][half][dV, dK][key][dim])
        if (ok && (nu == 0 || wait_all(B_FINAL, 0, 72))) {
            tc_fence_after();
            const bool isk = ch == 1;
            __nv_bfloat16 *dst = (isk ? prm.out0 : prm.out1) + ((size_t)(key < prm.T ? key : 0) * hkv + g) * kD;
            float *pdst = prm.split + ((((size_t)unit * hkv + g) * 2 + half) * 2 + (isk ? 1 : 0)) * (kKT * kD) +
                          (size_t)(lq * 32 + lane) * kD;
            const float mul = isk ? prm.scale : 1.f;
#pragma unroll
            for (int cc = 0; cc < 4; ++cc) {
                uint32_t o[32];
                if (nu > 0) {
                    tmem_ld32(tmem + lanes + (isk ? kColAcc1 : kColAcc0) + 32 * cc, o);
                    tmem_ld_wait();
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) o[i] = 0u;
                }
                if (split) {
#pragma unroll
                    for (int i = 0; i < 32; i += 4)
                        *reinterpret_cast<uint4 *>(pdst + 32 * cc + i) = make_uint4(o[i], o[i + 1], o[i + 2], o[i + 3]);
                } else if (key < prm.T) {
                    store_row_bf16(dst + 32 * cc, o, mul);
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// The split units' halves added (fp32), dK times scale, rounded once to bf16: one CTA per unit that
// may split (those that did not leave at once).
__global__ void __launch_bounds__(256) prefill_bwd_dkv_merge_kernel(const BwdParams prm)
{
    using namespace dkv;
    const int hkv = prm.num_kv_heads, group = prm.num_q_heads / hkv;
    const int unit = (int)(blockIdx.x / hkv), g = (int)(blockIdx.x % hkv);
    const int kt = prm.order[unit];
    const int ne = prm.ptr[kt + 1] - prm.ptr[kt];
    if (!(ne * group > PADOC_BWD_SPLIT_STEPS && unit < prm.split_units)) return;
    const float4 *p = reinterpret_cast<const float4 *>(prm.split + ((size_t)unit * hkv + g) * 4 * (kKT * kD));
    constexpr int kQuads = kKT * kD / 4;                  // float4 per tensor and half
    for (int x = threadIdx.x; x < 2 * kQuads; x += blockDim.x) {
        const int isk = x / kQuads, r = (x % kQuads) / (kD / 4), c4 = x % (kD / 4);
        const int64_t key = (int64_t)kt * kKT + r;
        if (key >= prm.T) continue;
        const float4 a = p[isk * kQuads + x % kQuads], b = p[(2 + isk) * kQuads + x % kQuads];
        const float mul = isk ? prm.scale : 1.f;
        uint2 w;
        w.x = pack_bf16x2((a.x + b.x) * mul, (a.y + b.y) * mul);
        w.y = pack_bf16x2((a.z + b.z) * mul, (a.w + b.w) * mul);
        *reinterpret_cast<uint2 *>((isk ? prm.out0 : prm.out1) + ((size_t)key * hkv + g) * kD + 4 * c4) = w;
    }
}

// ================================================================================================
// dQ pass
// ================================================================================================
// TMEM: Q at [0,64) and dO at [64,128) as A operands, the step buffers at 128 + 2W i (S, then dP),
// dQ at [384,512).
template <int W>
struct DqCfg {
    static constexpr int kQT = PADOC_BWD_DQ_Q_TILE;    // 128 query rows: the M of every MMA
    static constexpr int kDepth = 256 / (2 * W);
    static constexpr int kStages = W == 32 ? 8 : W == 64 ? 5 : 3;
    static constexpr int kPanel = W * 128;
    static constexpr int kTile = 2 * kPanel;            // K or V of one step
    static constexpr uint32_t kColQ = 0, kColG = 64, kColBuf = 128, kColDQ = 384;
    enum {
        B_QG = 0,                       // 256 arrivals: Q and dO stored into tensor memory
        B_KFULL = 1,                    // [stage]
        B_KEMPTY = 1 + kStages,         // [stage]
        B_SFULL = 1 + 2 * kStages,      // [buffer]
        B_PFULL = 1 + 2 * kStages + kDepth,   // [buffer], 256 arrivals
        B_FINAL = 1 + 2 * kStages + 2 * kDepth,
        B_COUNT = 2 + 2 * kStages + 2 * kDepth
    };
    static constexpr size_t kSmemBytes = 1024 + (size_t)kStages * 2 * kTile + B_COUNT * 8 + 64 + 2 * kQT * 4;
    static_assert(kDepth >= 1 && W % 32 == 0, "step width");
};

template <int W>
__global__ void __launch_bounds__(kThreads, 1)
prefill_bwd_dq_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                      const BwdParams prm)
{
    using C = DqCfg<W>;
    constexpr int S = C::kStages, DEPTH = C::kDepth;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *sk = smem;                        // [stage] K step tiles
    uint8_t *sv = sk + S * C::kTile;           // [stage] V step tiles
    uint64_t *bars = (uint64_t *)(sv + S * C::kTile);
    uint32_t *tmem_slot = (uint32_t *)(bars + C::B_COUNT);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    float *dsum = (float *)(tmem_slot + 16);   // [2][128]: the two column halves' parts of D

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int hq = prm.num_q_heads, group = hq / prm.num_kv_heads;
    const int qt = prm.num_tiles - 1 - (int)(blockIdx.x / hq);   // heavier q-tiles (later in a page) first
    const int h = (int)(blockIdx.x % hq), g = h / group;
    const int e0 = prm.ptr[qt], nu = prm.ptr[qt + 1] - e0;
    auto bar = [&](int i) { return smem_u32(&bars[i]); };

    if (tid == 0) {
        for (int i = 0; i < C::B_COUNT; ++i)
            mbar_init(bar(i), (i == C::B_QG || (i >= C::B_PFULL && i < C::B_PFULL + DEPTH)) ? 256 : 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 9) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 8) {
        // ---------------------------------------------------------------- TMA producer
        if (lane == 0 && nu > 0) {
            tma_prefetch_desc(&kmap);
            tma_prefetch_desc(&vmap);
            int issued = 0;
            for (int u = 0; u < nu; ++u) {
                const int s = u % S;
                if (u >= S && !wait_or_abort(bar(C::B_KEMPTY + s), (u / S - 1) & 1, prm.err, 80, abort_flag)) break;
                const int k0 = prm.idx[e0 + u] * W;
                const uint32_t fb = bar(C::B_KFULL + s);
                const uint32_t kb = smem_u32(sk + s * C::kTile), vb = smem_u32(sv + s * C::kTile);
                mbar_arrive_expect_tx(fb, 2 * C::kTile);
                tma_load_2d(kb, &kmap, g * kD, k0, fb);
                tma_load_2d(kb + C::kPanel, &kmap, g * kD + 64, k0, fb);
                tma_load_2d(vb, &vmap, g * kD, k0, fb);
                tma_load_2d(vb + C::kPanel, &vmap, g * kD + 64, k0, fb);
                issued = u + 1;
            }
            for (int u = (issued > S ? issued - S : 0); u < issued; ++u)
                mbar_wait_bounded(bar(C::B_KFULL + u % S), (u / S) & 1, prm.err, 82);
        }
    } else if (warp == 9) {
        // ---------------------------------------------------------------- MMA issuer (whole warp)
        if (nu > 0) {
            constexpr uint32_t idS = umma_idesc_bf16(128, W, false);
            constexpr uint32_t idAcc = umma_idesc_bf16(128, kD, true);
            auto wait_w = [&](int b, uint32_t parity, int site) {
                const bool r = wait_or_abort(bar(b), parity, prm.err, site, abort_flag);
                return __all_sync(0xffffffffu, r);
            };
            // S = Q K^T and dP = dO V^T of step u into buffer u % DEPTH (A from tensor memory)
            auto issue_s = [&](int u) {
                const int s = u % S;
                const uint32_t b = C::kColBuf + (uint32_t)(u % DEPTH) * 2 * W;
                if (!wait_w(C::B_KFULL + s, (u / S) & 1, 91)) return false;
                tc_fence_after();
                const uint64_t dk = umma_desc_sw128(smem_u32(sk + s * C::kTile), 16, 1024);
                const uint64_t dv = umma_desc_sw128(smem_u32(sv + s * C::kTile), 16, 1024);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    umma_bf16_ts_warp(tmem + b, tmem + C::kColQ + 8 * ks,
                                      dk + (((ks >> 2) * C::kPanel + (ks & 3) * 32) >> 4), idS, ks > 0);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    umma_bf16_ts_warp(tmem + b + W, tmem + C::kColG + 8 * ks,
                                      dv + (((ks >> 2) * C::kPanel + (ks & 3) * 32) >> 4), idS, ks > 0);
                umma_commit_warp(bar(C::B_SFULL + u % DEPTH));
                return true;
            };
            bool ok = wait_w(C::B_QG, 0, 90);
            if (ok) tc_fence_after();
            for (int u = 0; ok && u < DEPTH && u < nu; ++u) ok = issue_s(u);
            for (int u = 0; ok && u < nu; ++u) {
                const int s = u % S;
                const uint32_t b = C::kColBuf + (uint32_t)(u % DEPTH) * 2 * W;
                if (!wait_w(C::B_PFULL + u % DEPTH, (u / DEPTH) & 1, 92)) { ok = false; break; }
                tc_fence_after();
                // the step's K as an MN-major B operand (N = head dim, K = the W keys)
                const uint64_t kmn = umma_desc_sw128(smem_u32(sk + s * C::kTile), C::kPanel, 1024);
#pragma unroll
                for (int k = 0; k < W / 16; ++k)
                    umma_bf16_ts_warp(tmem + C::kColDQ, tmem + b + W + slice_col<W>(k), kmn + k * (2048 >> 4), idAcc,
                                      (u > 0 || k > 0));
                umma_commit_warp(bar(C::B_KEMPTY + s));
                if (u + DEPTH < nu && !issue_s(u + DEPTH)) { ok = false; break; }
            }
            umma_commit_warp(bar(C::B_FINAL));
            mbar_wait_bounded(bar(C::B_FINAL), 0, prm.err, 94);
        }
    } else {
        // ---------------------------------------------------------------- softmax + epilogue
        constexpr int HW = W / 2;
        const int lq = warp & 3, ch = warp >> 2;
        const int row = lq * 32 + lane;
        const int64_t t = (int64_t)qt * C::kQT + row;
        const uint32_t lanes = (uint32_t)(lq * 32) << 16;
        const float c = prm.scale_log2;
        int a0 = 0, a1 = 0, b0 = 0, b1 = 0;
        if (t < prm.T) {
            const int4 w = *reinterpret_cast<const int4 *>(prm.spans + 4 * t);
            a0 = w.x; a1 = w.y; b0 = w.z; b1 = w.w;
        }
        const uint64_t c2 = f2_pack(c, c);
        auto wait_all = [&](int b, uint32_t parity, int site) {
            const bool r = wait_or_abort(bar(b), parity, prm.err, site, abort_flag);
            return __all_sync(0xffffffffu, r);
        };
        // Q and dO rows of this query into tensor memory (dims 64 ch .. 64 ch + 63), and the row's
        // statistics: D = dO . O (fp32, the two column halves added through shared memory) and
        // -lse2; rows past T get -lse2 = -inf and D = 0, so that their P and dS are 0. Every
        // (row, head) of [0, t_pad) belongs to exactly one CTA, which writes them for the dK/dV pass.
        float nlrow, drow;
        {
            const bool in = t < prm.T;
            const size_t off = ((size_t)(in ? t : 0) * hq + h) * kD + 64 * ch;
            row_to_tmem(tmem + lanes + C::kColQ + 32 * ch, in ? prm.a0 + off : nullptr);
            uint32_t w[32];
            uint64_t acc2 = f2_pack(0.f, 0.f);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const uint4 x = in ? reinterpret_cast<const uint4 *>(prm.a1 + off)[i] : make_uint4(0u, 0u, 0u, 0u);
                const uint4 y = in ? reinterpret_cast<const uint4 *>(prm.o + off)[i] : make_uint4(0u, 0u, 0u, 0u);
                const uint32_t xs[4] = {x.x, x.y, x.z, x.w}, ys[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    w[4 * i + j] = xs[j];
                    acc2 = f2_fma(f2_pack(__uint_as_float(xs[j] << 16), __uint_as_float(xs[j] & 0xffff0000u)),
                                  f2_pack(__uint_as_float(ys[j] << 16), __uint_as_float(ys[j] & 0xffff0000u)), acc2);
                }
            }
            tmem_st32(tmem + lanes + C::kColG + 32 * ch, w);
            tmem_st_wait();
            tc_fence_before();
            mbar_arrive(bar(C::B_QG));
            float lo, hi;
            f2_unpack(acc2, lo, hi);
            dsum[ch * C::kQT + row] = lo + hi;
            named_bar_sync(1, 256);   // the eight softmax warps
            drow = dsum[row] + dsum[C::kQT + row];
            const float l = in ? prm.lse[(size_t)t * hq + h] : -INFINITY;
            nlrow = l == -INFINITY ? -INFINITY : -l * PADOC_LOG2E;
            if (!in) drow = 0.f;
            if (ch == 0) {
                prm.lt[(size_t)h * prm.t_pad + t] = nlrow;
                prm.dt[(size_t)h * prm.t_pad + t] = drow;
            }
        }
        const uint64_t nl2 = f2_pack(nlrow, nlrow), d2 = f2_pack(drow, drow);
        bool ok = true;
        for (int u = 0; u < nu; ++u) {
            const uint32_t b = C::kColBuf + (uint32_t)(u % DEPTH) * 2 * W + HW * ch;
            const bool partial = prm.kind[e0 + u] != PADOC_TILE_FULL;
            const int cb = prm.idx[e0 + u] * W + HW * ch;
            if (!wait_all(C::B_SFULL + u % DEPTH, (u / DEPTH) & 1, 95)) { ok = false; break; }
            tc_fence_after();
            // the thread's HW key columns in blocks of at most 32: block j's dS (bf16 pairs) goes to
            // columns 16 j .. of its half of the dP buffer, which block j has already read
            constexpr int HB = HW < 32 ? HW : 32;
#pragma unroll
            for (int j = 0; j < HW / HB; ++j) {
                uint32_t sr[HB], dr[HB];
                tmem_ld_cols<HB>(tmem + lanes + b + HB * j, sr);
                tmem_ld_cols<HB>(tmem + lanes + b + W + HB * j, dr);
                uint32_t vis = 0xffffffffu;
                if (partial) {
                    const int cj = cb + HB * j;
                    const int lo0 = clamp_w(a0 - cj, HB), lo1 = clamp_w(b0 - cj, HB);
                    vis = interval_bits(lo0, max(clamp_w(a1 - cj, HB) - lo0, 0), 0) |
                          interval_bits(lo1, max(clamp_w(b1 - cj, HB) - lo1, 0), 0);
                }
                tmem_ld_wait();
                uint32_t dk[HB / 2];
                // two key columns per packed instruction: P = exp2(S c - lse2), dS = P (dP - D)
                auto column_pairs = [&](auto masked) {
#pragma unroll
                    for (int i = 0; i < HB; i += 2) {
                        float x0, x1;
                        f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[i]), __uint_as_float(sr[i + 1])), c2, nl2), x0, x1);
                        float p0 = fast_exp2(x0), p1 = fast_exp2(x1);
                        if (decltype(masked)::value) {
                            p0 = (vis >> i) & 1u ? p0 : 0.f;
                            p1 = (vis >> (i + 1)) & 1u ? p1 : 0.f;
                        }
                        const uint64_t t = f2_sub(f2_pack(__uint_as_float(dr[i]), __uint_as_float(dr[i + 1])), d2);
                        float d0, d1;
                        f2_unpack(f2_mul(f2_pack(p0, p1), t), d0, d1);
                        dk[i >> 1] = pack_bf16x2(d0, d1);
                    }
                };
                if (partial) column_pairs(std::true_type{}); else column_pairs(std::false_type{});
                tmem_st_cols<HB / 2>(tmem + lanes + b + W + (HB / 2) * j, dk);
            }
            tmem_st_wait();
            tc_fence_before();
            mbar_arrive(bar(C::B_PFULL + u % DEPTH));
        }
        // epilogue: dQ times scale, columns 64 ch .. 64 ch + 63 of the thread's row
        if (ok && (nu == 0 || wait_all(C::B_FINAL, 0, 96))) {
            tc_fence_after();
            __nv_bfloat16 *dst = prm.out0 + ((size_t)(t < prm.T ? t : 0) * hq + h) * kD + 64 * ch;
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                uint32_t o[32];
                if (nu > 0) {
                    tmem_ld32(tmem + lanes + C::kColDQ + 64 * ch + 32 * cc, o);
                    tmem_ld_wait();
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) o[i] = 0u;
                }
                if (t < prm.T) store_row_bf16(dst + 32 * cc, o, prm.scale);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

padoc_status padoc_launch_prefill_bwd_tc(const void *q, const void *k, const void *v, const void *out,
                                         const void *dout, const float *lse, int64_t total_tokens,
                                         int32_t num_q_heads, int32_t num_kv_heads, const int32_t *spans_dev,
                                         const padoc_tile_map_dev *q_map, const padoc_tile_map_dev *k_map, float *lt,
                                         float *dt, float *split, int64_t t_pad, float scale, void *dq, void *dk,
                                         void *dv, cudaStream_t stream)
{
    constexpr int WQ = PADOC_BWD_DQ_K_TILE;
    using CQ = DqCfg<WQ>;
    int *err = padoc_device_error_word();
    if (!err) return PADOC_ERR_CUDA;
    const int64_t T = total_tokens;
    const int64_t nkt = (T + dkv::kKT - 1) / dkv::kKT, nqt = (T + CQ::kQT - 1) / CQ::kQT;
    if (2 * nkt * num_kv_heads > INT32_MAX || nqt * num_q_heads > INT32_MAX) return PADOC_ERR_UNSUPPORTED;
    const uint64_t qcols = (uint64_t)num_q_heads * kD, kcols = (uint64_t)num_kv_heads * kD;
    CUtensorMap q64, g64, k128, v128, kmap, vmap;
    if (!padoc_make_tmap_bf16(&q64, q, qcols, T, qcols * 2, 64, dkv::kQT) ||
        !padoc_make_tmap_bf16(&g64, dout, qcols, T, qcols * 2, 64, dkv::kQT) ||
        !padoc_make_tmap_bf16(&k128, k, kcols, T, kcols * 2, 64, dkv::kKT) ||
        !padoc_make_tmap_bf16(&v128, v, kcols, T, kcols * 2, 64, dkv::kKT) ||
        !padoc_make_tmap_bf16(&kmap, k, kcols, T, kcols * 2, 64, WQ) ||
        !padoc_make_tmap_bf16(&vmap, v, kcols, T, kcols * 2, 64, WQ))
        return PADOC_ERR_CUDA;
    BwdParams prm;
    prm.spans = spans_dev;
    prm.lt = lt;
    prm.dt = dt;
    prm.T = T;
    prm.t_pad = t_pad;
    prm.num_q_heads = num_q_heads;
    prm.num_kv_heads = num_kv_heads;
    prm.scale_log2 = scale * PADOC_LOG2E;
    prm.scale = scale;
    prm.err = err;
    prm.o = nullptr;
    prm.lse = nullptr;
    prm.split = split;
    // the units that may split: their partials (2 halves x 2 tensors x 64 KB per KV head) fit in the
    // workspace's PADOC_BWD_SPLIT_BYTES_PER_TOKEN bytes per token of t_pad
    prm.split_units = (int32_t)std::min<int64_t>(nkt, t_pad * PADOC_BWD_SPLIT_BYTES_PER_TOKEN /
                                                          ((int64_t)num_kv_heads * 4 * dkv::kKT * kD * 4));

    // the dQ pass first: it also writes -lse2 and D of every row for the dK/dV pass
    BwdParams pq = prm;   // dQ pass over the query-major map; Q and dO go to tensor memory
    pq.ptr = q_map->ptr;
    pq.idx = q_map->idx;
    pq.kind = q_map->kind;
    pq.order = nullptr;
    pq.a0 = (const __nv_bfloat16 *)q;
    pq.a1 = (const __nv_bfloat16 *)dout;
    pq.num_tiles = (int32_t)nqt;
    pq.out0 = (__nv_bfloat16 *)dq;
    pq.out1 = nullptr;
    pq.o = (const __nv_bfloat16 *)out;
    pq.lse = lse;
    PADOC_CUDA_TRY(cudaFuncSetAttribute(prefill_bwd_dq_kernel<WQ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        (int)CQ::kSmemBytes));
    prefill_bwd_dq_kernel<WQ><<<(unsigned)(nqt * num_q_heads), kThreads, CQ::kSmemBytes, stream>>>(kmap, vmap, pq);
    padoc_status st = padoc_launch_status();
    if (st != PADOC_OK) return st;

    BwdParams pk = prm;   // dK/dV pass over the key-major map
    pk.ptr = k_map->ptr;
    pk.idx = k_map->idx;
    pk.kind = k_map->kind;
    pk.order = k_map->order;
    pk.num_tiles = (int32_t)nkt;
    pk.out0 = (__nv_bfloat16 *)dk;
    pk.out1 = (__nv_bfloat16 *)dv;
    PADOC_CUDA_TRY(cudaFuncSetAttribute(prefill_bwd_dkv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        (int)dkv::kSmemBytes));
    prefill_bwd_dkv_kernel<<<(unsigned)(2 * nkt * num_kv_heads), kThreads, dkv::kSmemBytes, stream>>>(q64, g64, k128,
                                                                                                       v128, pk);
    st = padoc_launch_status();
    if (st != PADOC_OK || pk.split_units == 0) return st;
    prefill_bwd_dkv_merge_kernel<<<(unsigned)(pk.split_units * num_kv_heads), 256, 0, stream>>>(pk);
    return padoc_launch_status();
}
