// prefill_tc.cu -- C3 on the 5th-generation tensor cores: packed variable-length ancestor prefill
// (App. C.1: the causal problem over M and one bottom-right-aligned causal problem per branch over
// [K_{M<=f_k}; K_{Y_k}], computed in packed order without a gather).
//
// One CTA per (128-row q-tile, pair of query heads sharing a KV head); with an odd GQA group the
// CTA takes one head. It walks the q-tile's entries of the tile map: fully masked k-tiles are never
// visited, FULL tiles skip masking, PARTIAL tiles mask each row with its two spans. The two heads
// share every K/V tile the producer stages, and their softmax warpgroups alternate with the tensor
// core (while one warpgroup exponentiates, the MMAs of the other head run).
//
// Warp roles (320 threads):
//   warps 0-3 / 4-7  softmax + epilogue of head 0 / head 1; thread t owns query row t (TMEM lane
//                    t), so row max and row sum need no shuffles;
//   warp 8           TMA producer: both heads' Q once, then K and V tiles (128 keys x 128 dims,
//                    two 64-column panels each, 128-byte swizzle) into a 2-stage ring;
//   warp 9           TMEM allocation and the MMA issuer (one thread).
// TMEM (512 columns): head i keeps S_i at columns 128i..128i+127 and O_i at 256+128i. The softmax
// writes P_i as packed bf16 over the first 64 columns of S_i, and O_i += P_i V reads P_i straight
// from TMEM (V as an MN-major shared-memory operand). For head i the MMAs run S_i(j) -> P_i(j) ->
// PV_i(j) -> S_i(j+1) in issue order, so S_i(j+1) never overwrites a P_i still being read.
// O is rescaled lazily: the reference maximum only moves when a row's maximum grows by more than
// 2^8, which keeps every P entry <= 256 and the arithmetic exact up to rounding.
// Every wait is bounded; a wait that runs out records an error, all roles leave their loops, the
// MMA issuer waits for its MMAs, the producer for its copies, and TMEM is released.
#include <math.h>

#include "common.cuh"
#include "tc.cuh"

namespace {

constexpr int kD = 128;
constexpr int kQT = PADOC_PREFILL_Q_TILE;
constexpr int kKT = PADOC_PREFILL_K_TILE;
constexpr int kPanel = 128 * 128;    // [128 rows][64 bf16]
constexpr int kTile = 2 * kPanel;    // 32 KB
constexpr int kStages = 2;
constexpr uint32_t kTmemCols = 512;
constexpr int kThreads = 320;

enum {
    B_Q = 0,
    B_KFULL = 1,     // [stage]
    B_VFULL = 3,     // [stage]
    B_KVEMPTY = 5,   // [stage]
    B_SFULL = 7,     // [head]
    B_PFULL = 9,     // [head], 128 arrivals
    B_PVDONE = 11,   // [head]
    B_FINAL = 13,
    B_COUNT = 14
};

constexpr size_t kSmemBytes = 1024 + (size_t)kTile * (2 + 2 * kStages) + B_COUNT * 8 + 64;

struct TcPrefillParams {
    const int32_t *spans, *row_ptr, *tile_k;
    const int8_t *tile_kind;
    int64_t T;
    int32_t num_q_heads, num_kv_heads, num_q_tiles, heads_per_cta;
    float scale_log2;
    __nv_bfloat16 *out;
    float *lse;
    int *err;
};

__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, int *err, int site, volatile int *abort_flag)
{
    if (*abort_flag) return false;
    if (mbar_wait_bounded(bar, parity, err, site)) return true;
    *abort_flag = 1;
    return false;
}

__device__ __forceinline__ int clamp_tile(int x) { return min(max(x, 0), kKT); }

template <int NH>
__global__ void __launch_bounds__(kThreads, 1)
prefill_tc_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                  const __grid_constant__ CUtensorMap vmap, const TcPrefillParams prm)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *sq = smem;                       // [2 heads] tiles
    uint8_t *sk = sq + 2 * kTile;             // [kStages] tiles
    uint8_t *sv = sk + kStages * kTile;       // [kStages] tiles
    uint64_t *bars = (uint64_t *)(sv + kStages * kTile);
    uint32_t *tmem_slot = (uint32_t *)(bars + B_COUNT);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    constexpr int nh = NH;
    const int h0 = blockIdx.x * nh;
    const int qt = prm.num_q_tiles - 1 - (int)blockIdx.y;   // heavier tiles (later in a page) first
    const int g = h0 / (prm.num_q_heads / prm.num_kv_heads);
    const int e0 = prm.row_ptr[qt], ne = prm.row_ptr[qt + 1] - e0;
    auto bar = [&](int i) { return smem_u32(&bars[i]); };

    if (tid == 0) {
        for (int i = 0; i < B_COUNT; ++i) mbar_init(bar(i), (i == B_PFULL || i == B_PFULL + 1) ? 128 : 1);
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
        if (lane == 0 && ne > 0) {
            tma_prefetch_desc(&qmap);
            tma_prefetch_desc(&kmap);
            tma_prefetch_desc(&vmap);
            mbar_arrive_expect_tx(bar(B_Q), nh * kTile);
            for (int i = 0; i < nh; ++i) {
                tma_load_2d(smem_u32(sq + i * kTile), &qmap, (h0 + i) * kD, qt * kQT, bar(B_Q));
                tma_load_2d(smem_u32(sq + i * kTile) + kPanel, &qmap, (h0 + i) * kD + 64, qt * kQT, bar(B_Q));
            }
            int issued = 0;
            for (int j = 0; j < ne; ++j) {
                const int s = j & 1;
                if (j >= 2 && !wait_or_abort(bar(B_KVEMPTY + s), ((j - 2) >> 1) & 1, prm.err, 20, abort_flag)) break;
                const int kt = prm.tile_k[e0 + j];
                const uint32_t kb = smem_u32(sk + s * kTile), vb = smem_u32(sv + s * kTile);
                mbar_arrive_expect_tx(bar(B_KFULL + s), kTile);
                tma_load_2d(kb, &kmap, g * kD, kt * kKT, bar(B_KFULL + s));
                tma_load_2d(kb + kPanel, &kmap, g * kD + 64, kt * kKT, bar(B_KFULL + s));
                mbar_arrive_expect_tx(bar(B_VFULL + s), kTile);
                tma_load_2d(vb, &vmap, g * kD, kt * kKT, bar(B_VFULL + s));
                tma_load_2d(vb + kPanel, &vmap, g * kD + 64, kt * kKT, bar(B_VFULL + s));
                issued = j + 1;
            }
            // copies still in flight must land before the CTA's shared memory is released
            mbar_wait_bounded(bar(B_Q), 0, prm.err, 21);
            for (int j = (issued > 2 ? issued - 2 : 0); j < issued; ++j) {
                mbar_wait_bounded(bar(B_KFULL + (j & 1)), (j >> 1) & 1, prm.err, 22);
                mbar_wait_bounded(bar(B_VFULL + (j & 1)), (j >> 1) & 1, prm.err, 23);
            }
        }
    } else if (warp == 9) {
        // ---------------------------------------------------------------- MMA issuer (whole warp)
        if (ne > 0) {
            constexpr uint32_t idS = umma_idesc_bf16(128, kKT, false);
            constexpr uint32_t idPV = umma_idesc_bf16(128, kD, true);
            // descriptor bases; a K-step adds a constant to the 14-bit start-address field
            // (addresses stay below 256 KB, so the field never carries)
            const uint64_t dq0 = umma_desc_sw128(smem_u32(sq), 16, 1024);
            const uint64_t dq1 = umma_desc_sw128(smem_u32(sq + kTile), 16, 1024);
            const uint64_t dk0 = umma_desc_sw128(smem_u32(sk), 16, 1024);
            const uint64_t dk1 = umma_desc_sw128(smem_u32(sk + kTile), 16, 1024);
            const uint64_t dv0 = umma_desc_sw128(smem_u32(sv), kPanel, 1024);
            const uint64_t dv1 = umma_desc_sw128(smem_u32(sv + kTile), kPanel, 1024);
            auto wait_w = [&](int b, uint32_t parity, int site) {
                const bool r = wait_or_abort(bar(b), parity, prm.err, site, abort_flag);
                return __all_sync(0xffffffffu, r);
            };
            auto issue_s = [&](int i, int stage) {
                const uint64_t da = i ? dq1 : dq0, db = stage ? dk1 : dk0;
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {
                    const uint32_t off = ((ks >> 2) * kPanel + (ks & 3) * 32) >> 4;
                    umma_bf16_ss_warp(tmem + 128 * i, da + off, db + off, idS, ks > 0);
                }
                umma_commit_warp(bar(B_SFULL + i));
            };
            bool ok = wait_w(B_Q, 0, 30) && wait_w(B_KFULL, 0, 31);
            if (ok) {
                tc_fence_after();
#pragma unroll
                for (int i = 0; i < NH; ++i) issue_s(i, 0);
            }
            for (int j = 0; ok && j < ne; ++j) {
                const int s = j & 1, sn = (j + 1) & 1;
#pragma unroll
                for (int i = 0; i < NH; ++i) {
                    if (!wait_w(B_PFULL + i, j & 1, 32)) { ok = false; break; }
                    if (i == 0 && !wait_w(B_VFULL + s, (j >> 1) & 1, 33)) { ok = false; break; }
                    tc_fence_after();
                    const uint64_t db = s ? dv1 : dv0;
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk)
                        umma_bf16_ts_warp(tmem + 256 + 128 * i, tmem + 128 * i + kk * 8, db + kk * (2048 >> 4), idPV,
                                          (j > 0 || kk > 0));
                    umma_commit_warp(bar(B_PVDONE + i));
                    if (i == NH - 1) umma_commit_warp(bar(B_KVEMPTY + s));
                    if (j + 1 < ne) {
                        if (i == 0 && !wait_w(B_KFULL + sn, ((j + 1) >> 1) & 1, 34)) { ok = false; break; }
                        tc_fence_after();
                        issue_s(i, sn);
                    }
                }
            }
            // every MMA issued above must complete before TMEM is released
            umma_commit_warp(bar(B_FINAL));
            mbar_wait_bounded(bar(B_FINAL), 0, prm.err, 35);
        }
    } else if (warp / 4 < nh) {
        // ---------------------------------------------------------------- softmax + epilogue
        const int hi = warp / 4;                    // head index inside the CTA
        const int h = h0 + hi;
        const int row = tid & 127;
        const int64_t t = (int64_t)qt * kQT + row;
        int a0 = 0, a1 = 0, b0 = 0, b1 = 0;
        if (t < prm.T) {
            const int4 v = *reinterpret_cast<const int4 *>(prm.spans + 4 * t);
            a0 = v.x; a1 = v.y; b0 = v.z; b1 = v.w;
        }
        const uint32_t lanes = (uint32_t)((warp & 3) * 32) << 16;
        const uint32_t tS = tmem + lanes + 128 * hi, tO = tmem + lanes + 256 + 128 * hi;
        const float c = prm.scale_log2;
        // every decision below is warp-uniform: the TMEM loads and stores are warp-collective
        auto wait_all = [&](int b, uint32_t parity, int site) {
            const bool r = wait_or_abort(bar(b), parity, prm.err, site, abort_flag);
            return __all_sync(0xffffffffu, r);
        };
        float m_ref = -INFINITY, l = 0.f;   // m_ref in raw score units
        bool ok = ne > 0;
        int kt_next = ne > 0 ? prm.tile_k[e0] : 0, kind_next = ne > 0 ? prm.tile_kind[e0] : 0;
        for (int j = 0; ok && j < ne; ++j) {
            const int kt = kt_next;
            const bool full = kind_next == PADOC_TILE_FULL;   // the same for every row of the CTA
            if (j + 1 < ne) { kt_next = prm.tile_k[e0 + j + 1]; kind_next = prm.tile_kind[e0 + j + 1]; }
            if (!wait_all(B_SFULL + hi, j & 1, 40)) { ok = false; break; }
            tc_fence_after();
            // pass 1: row maximum, 32 columns at a time; a PARTIAL tile also writes its masked
            // scores back so that pass 2 reads them unmasked
            float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
            if (full) {
#pragma unroll
                for (int q = 0; q < 4; q += 2) {
                    uint32_t sr[2][32];
                    tmem_ld32(tS + q * 32, sr[0]);
                    tmem_ld32(tS + q * 32 + 32, sr[1]);
                    tmem_ld_wait();
#pragma unroll
                    for (int u = 0; u < 2; ++u)
#pragma unroll
                        for (int i = 0; i < 32; i += 8) {
                            mx4[0] = fmax3f(mx4[0], __uint_as_float(sr[u][i]), __uint_as_float(sr[u][i + 1]));
                            mx4[1] = fmax3f(mx4[1], __uint_as_float(sr[u][i + 2]), __uint_as_float(sr[u][i + 3]));
                            mx4[2] = fmax3f(mx4[2], __uint_as_float(sr[u][i + 4]), __uint_as_float(sr[u][i + 5]));
                            mx4[3] = fmax3f(mx4[3], __uint_as_float(sr[u][i + 6]), __uint_as_float(sr[u][i + 7]));
                        }
                }
            } else {
                const int cb = kt * kKT;
                const int lo0 = clamp_tile(a0 - cb), w0 = max(clamp_tile(a1 - cb) - lo0, 0);
                const int lo1 = clamp_tile(b0 - cb), w1 = max(clamp_tile(b1 - cb) - lo1, 0);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint32_t vis = interval_bits(lo0, w0, q * 32) | interval_bits(lo1, w1, q * 32);
                    uint32_t sr[32];
                    tmem_ld32(tS + q * 32, sr);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i) sr[i] = (vis >> i) & 1u ? sr[i] : 0xff800000u;   // -inf
#pragma unroll
                    for (int i = 0; i < 32; i += 8) {
                        mx4[0] = fmax3f(mx4[0], __uint_as_float(sr[i]), __uint_as_float(sr[i + 1]));
                        mx4[1] = fmax3f(mx4[1], __uint_as_float(sr[i + 2]), __uint_as_float(sr[i + 3]));
                        mx4[2] = fmax3f(mx4[2], __uint_as_float(sr[i + 4]), __uint_as_float(sr[i + 5]));
                        mx4[3] = fmax3f(mx4[3], __uint_as_float(sr[i + 6]), __uint_as_float(sr[i + 7]));
                    }
                    tmem_st32(tS + q * 32, sr);
                }
                tmem_st_wait();
            }
            const float mx = fmaxf(fmax3f(mx4[0], mx4[1], mx4[2]), mx4[3]);
            const float m_new = fmaxf(m_ref, mx);
            // a row with nothing accumulated yet (O holds zeros) adopts the new maximum directly;
            // otherwise the reference only moves when the maximum grew by more than 2^8
            const bool rescale = m_ref != -INFINITY && (m_new - m_ref) * c > 8.f;
            if (m_ref == -INFINITY) m_ref = m_new;
            if (__any_sync(0xffffffffu, rescale)) {
                // PV_i(j-1) completed before S_i(j) (issue order), so O_i is quiescent here
                const float alpha = rescale ? fast_exp2((m_ref - m_new) * c) : 1.f;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint32_t o[32];
                    tmem_ld32(tO + q * 32, o);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                    tmem_st32(tO + q * 32, o);
                }
                if (rescale) { l *= alpha; m_ref = m_new; }
            }
            const float moff = m_ref == -INFINITY ? 0.f : m_ref * c;
            // pass 2: P = exp2(S * c - m * c) as packed bf16 over the first 64 columns of S
            float rs[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                uint32_t pk[32];
                uint32_t sr[2][32];
                tmem_ld32(tS + half * 64, sr[0]);
                tmem_ld32(tS + half * 64 + 32, sr[1]);
                tmem_ld_wait();
#pragma unroll
                for (int qq = 0; qq < 2; ++qq) {
#pragma unroll
                    for (int i = 0; i < 32; i += 2) {
                        const float p0 = fast_exp2(fmaf(__uint_as_float(sr[qq][i]), c, -moff));
                        const float p1 = fast_exp2(fmaf(__uint_as_float(sr[qq][i + 1]), c, -moff));
                        rs[(i >> 1) & 3] += p0 + p1;
                        pk[qq * 16 + (i >> 1)] = pack_bf16x2(p0, p1);
                    }
                }
                tmem_st32(tS + half * 32, pk);
            }
            l += (rs[0] + rs[1]) + (rs[2] + rs[3]);
            tmem_st_wait();
            tc_fence_before();
            mbar_arrive(bar(B_PFULL + hi));
        }
        if (ok && wait_all(B_PVDONE + hi, (ne - 1) & 1, 43)) {
            tc_fence_after();
            const float inv = l > 0.f ? 1.f / l : 0.f;
            __nv_bfloat16 *orow = prm.out + ((size_t)(t < prm.T ? t : 0) * prm.num_q_heads + h) * kD;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                uint32_t o[32];
                tmem_ld32(tO + q * 32, o);
                tmem_ld_wait();
                if (t < prm.T) {
#pragma unroll
                    for (int i = 0; i < 32; i += 8) {
                        uint4 w;
                        w.x = pack_bf16x2(__uint_as_float(o[i]) * inv, __uint_as_float(o[i + 1]) * inv);
                        w.y = pack_bf16x2(__uint_as_float(o[i + 2]) * inv, __uint_as_float(o[i + 3]) * inv);
                        w.z = pack_bf16x2(__uint_as_float(o[i + 4]) * inv, __uint_as_float(o[i + 5]) * inv);
                        w.w = pack_bf16x2(__uint_as_float(o[i + 6]) * inv, __uint_as_float(o[i + 7]) * inv);
                        *reinterpret_cast<uint4 *>(orow + q * 32 + i) = w;
                    }
                }
            }
            if (t < prm.T)
                prm.lse[(size_t)t * prm.num_q_heads + h] = l > 0.f ? (m_ref * c + log2f(l)) * PADOC_LN2 : -INFINITY;
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

padoc_status padoc_launch_prefill_tc(const void *q, const void *k, const void *v, int64_t total_tokens,
                                     int32_t num_q_heads, int32_t num_kv_heads, const int32_t *spans_dev,
                                     const int32_t *tile_row_ptr_dev, const int32_t *tile_k_dev,
                                     const int8_t *tile_kind_dev, float scale_log2, void *out, float *lse,
                                     cudaStream_t stream)
{
    int *err = padoc_device_error_word();
    if (!err) return PADOC_ERR_CUDA;
    const int64_t nqt = (total_tokens + kQT - 1) / kQT;
    if (nqt > 65535) return PADOC_ERR_UNSUPPORTED;
    CUtensorMap qmap, kmap, vmap;
    if (!padoc_make_tmap_bf16(&qmap, q, (uint64_t)num_q_heads * kD, total_tokens, (uint64_t)num_q_heads * kD * 2, 64, kQT) ||
        !padoc_make_tmap_bf16(&kmap, k, (uint64_t)num_kv_heads * kD, total_tokens, (uint64_t)num_kv_heads * kD * 2, 64, kKT) ||
        !padoc_make_tmap_bf16(&vmap, v, (uint64_t)num_kv_heads * kD, total_tokens, (uint64_t)num_kv_heads * kD * 2, 64, kKT))
        return PADOC_ERR_CUDA;
    TcPrefillParams prm;
    prm.spans = spans_dev;
    prm.row_ptr = tile_row_ptr_dev;
    prm.tile_k = tile_k_dev;
    prm.tile_kind = tile_kind_dev;
    prm.T = total_tokens;
    prm.num_q_heads = num_q_heads;
    prm.num_kv_heads = num_kv_heads;
    prm.num_q_tiles = (int32_t)nqt;
    prm.heads_per_cta = ((num_q_heads / num_kv_heads) % 2 == 0) ? 2 : 1;   // a pair must share its KV head
    prm.scale_log2 = scale_log2;
    prm.out = (__nv_bfloat16 *)out;
    prm.lse = lse;
    prm.err = err;
    dim3 grid((unsigned)(num_q_heads / prm.heads_per_cta), (unsigned)nqt);
    if (prm.heads_per_cta == 2) {
        PADOC_CUDA_TRY(cudaFuncSetAttribute(prefill_tc_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes));
        prefill_tc_kernel<2><<<grid, kThreads, kSmemBytes, stream>>>(qmap, kmap, vmap, prm);
    } else {
        PADOC_CUDA_TRY(cudaFuncSetAttribute(prefill_tc_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes));
        prefill_tc_kernel<1><<<grid, kThreads, kSmemBytes, stream>>>(qmap, kmap, vmap, prm);
    }
    return padoc_launch_status();
}
