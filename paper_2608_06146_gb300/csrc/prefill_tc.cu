// prefill_tc.cu -- C3 on the 5th-generation tensor cores: packed variable-length ancestor prefill
// (App. C.1: the causal problem over M and one bottom-right-aligned causal problem per branch over
// [K_{M<=f_k}; K_{Y_k}], computed in packed order without a gather).
//
// One CTA per (128-row q-tile, query head), walking the q-tile's entries of the tile map (fully
// masked k-tiles are never visited; FULL tiles skip masking; PARTIAL tiles mask each row with its
// two spans). Warp roles:
//   warps 0-3  softmax + epilogue; thread t owns query row t (TMEM lane t), so row max and row sum
//              need no shuffles;
//   warp 4     TMA producer: Q once, then K and V tiles (128 keys x 128 dims, two 64-column
//              panels each, 128-byte swizzle) into a 2-stage ring;
//   warp 5     TMEM allocation and the MMA issuer (one thread).
// TMEM (512 columns): S double-buffered at columns 0 and 128 (so S_{j+1} = Q K_{j+1}^T runs on the
// tensor cores while the softmax of tile j runs), O at column 256. P is written as bf16 into a
// 128-byte-swizzled K-major shared-memory tile and consumed by O += P V (V as an MN-major operand).
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
constexpr uint32_t kColO = 256;

enum {
    B_Q = 0,
    B_KFULL = 1,     // [2]
    B_VFULL = 3,     // [2]
    B_KVEMPTY = 5,   // [2]
    B_SFULL = 7,     // [2]
    B_SFREE = 9,     // [2]
    B_PFULL = 11,
    B_PVDONE = 12,
    B_FINAL = 13,
    B_COUNT = 14
};

constexpr size_t kSmemBytes = 1024 + (size_t)kTile * (1 + 2 * kStages + 1) + B_COUNT * 8 + 64;

struct TcPrefillParams {
    const int32_t *spans, *row_ptr, *tile_k;
    const int8_t *tile_kind;
    int64_t T;
    int32_t num_q_heads, num_kv_heads, num_q_tiles;
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

__global__ void __launch_bounds__(192, 1)
prefill_tc_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                  const __grid_constant__ CUtensorMap vmap, const TcPrefillParams prm)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *sq = smem;
    uint8_t *sk = sq + kTile;                 // [kStages] tiles
    uint8_t *sv = sk + kStages * kTile;       // [kStages] tiles
    uint8_t *sp = sv + kStages * kTile;       // P
    uint64_t *bars = (uint64_t *)(sp + kTile);
    uint32_t *tmem_slot = (uint32_t *)(bars + B_COUNT);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int h = blockIdx.x;
    const int qt = prm.num_q_tiles - 1 - (int)blockIdx.y;
    const int g = h / (prm.num_q_heads / prm.num_kv_heads);
    const int e0 = prm.row_ptr[qt], ne = prm.row_ptr[qt + 1] - e0;
    auto bar = [&](int i) { return smem_u32(&bars[i]); };

    if (tid == 0) {
        for (int i = 0; i < B_COUNT; ++i) {
            const int cnt = (i == B_SFREE || i == B_SFREE + 1 || i == B_PFULL) ? 128 : 1;
            mbar_init(bar(i), cnt);
        }
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 5) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 4) {
        // ---------------------------------------------------------------- TMA producer
        if (lane == 0 && ne > 0) {
            tma_prefetch_desc(&qmap);
            tma_prefetch_desc(&kmap);
            tma_prefetch_desc(&vmap);
            mbar_arrive_expect_tx(bar(B_Q), kTile);
            tma_load_2d(smem_u32(sq), &qmap, h * kD, qt * kQT, bar(B_Q));
            tma_load_2d(smem_u32(sq) + kPanel, &qmap, h * kD + 64, qt * kQT, bar(B_Q));
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
    } else if (warp == 5) {
        // ---------------------------------------------------------------- MMA issuer
        if (lane == 0 && ne > 0) {
            const uint32_t idS = umma_idesc_bf16(128, kKT, false);
            const uint32_t idPV = umma_idesc_bf16(128, kD, true);
            const uint32_t uq = smem_u32(sq), up = smem_u32(sp);
            bool ok = wait_or_abort(bar(B_Q), 0, prm.err, 30, abort_flag);
            for (int j = 0; ok && j <= ne; ++j) {
                if (j < ne) {
                    const int s = j & 1;
                    if (!wait_or_abort(bar(B_KFULL + s), (j >> 1) & 1, prm.err, 31, abort_flag)) break;
                    if (j >= 2 && !wait_or_abort(bar(B_SFREE + s), ((j - 2) >> 1) & 1, prm.err, 32, abort_flag)) break;
                    tc_fence_after();
                    const uint32_t ub = smem_u32(sk + s * kTile);
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks) {
                        const uint32_t off = (ks >> 2) * kPanel + (ks & 3) * 32;
                        umma_bf16_ss(tmem + s * 128, umma_desc_sw128(uq + off, 16, 1024),
                                     umma_desc_sw128(ub + off, 16, 1024), idS, ks > 0);
                    }
                    umma_commit(bar(B_SFULL + s));
                }
                if (j >= 1) {
                    const int jp = j - 1, s = jp & 1;
                    if (!wait_or_abort(bar(B_PFULL), jp & 1, prm.err, 33, abort_flag)) break;
                    if (!wait_or_abort(bar(B_VFULL + s), (jp >> 1) & 1, prm.err, 34, abort_flag)) break;
                    tc_fence_after();
                    const uint32_t uv = smem_u32(sv + s * kTile);
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk) {
                        const uint32_t aoff = (kk >> 2) * kPanel + (kk & 3) * 32;
                        umma_bf16_ss(tmem + kColO, umma_desc_sw128(up + aoff, 16, 1024),
                                     umma_desc_sw128(uv + kk * 2048, kPanel, 1024), idPV, (jp > 0 || kk > 0));
                    }
                    umma_commit(bar(B_PVDONE));
                    umma_commit(bar(B_KVEMPTY + s));
                }
            }
            // every MMA issued above must complete before TMEM is released
            umma_commit(bar(B_FINAL));
            mbar_wait_bounded(bar(B_FINAL), 0, prm.err, 35);
        }
    } else {
        // ---------------------------------------------------------------- softmax + epilogue
        const int row = tid;
        const int64_t t = (int64_t)qt * kQT + row;
        int a0 = 0, a1 = 0, b0 = 0, b1 = 0;
        if (t < prm.T) {
            const int4 v = *reinterpret_cast<const int4 *>(prm.spans + 4 * t);
            a0 = v.x; a1 = v.y; b0 = v.z; b1 = v.w;
        }
        const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
        // every decision below is warp-uniform: the TMEM loads and stores are warp-collective
        auto wait_all = [&](int b, uint32_t parity, int site) {
            const bool r = wait_or_abort(bar(b), parity, prm.err, site, abort_flag);
            return __all_sync(0xffffffffu, r);
        };
        float m_ref = -INFINITY, l = 0.f;
        bool ok = ne > 0;
        for (int j = 0; ok && j < ne; ++j) {
            const int s = j & 1;
            if (!wait_all(B_SFULL + s, (j >> 1) & 1, 40)) { ok = false; break; }
            tc_fence_after();
            uint32_t sr[4][32];
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(lane_base + s * 128 + c * 32, sr[c]);
            tmem_ld_wait();
            tc_fence_before();
            mbar_arrive(bar(B_SFREE + s));

            const int kt = prm.tile_k[e0 + j];
            const bool full = prm.tile_kind[e0 + j] == PADOC_TILE_FULL;
            const int cbase = kt * kKT;
            float mx = -INFINITY;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    float x = __uint_as_float(sr[c][i]) * prm.scale_log2;
                    if (!full) {
                        const int jj = cbase + c * 32 + i;
                        const bool vis = (jj >= a0 && jj < a1) || (jj >= b0 && jj < b1);
                        x = vis ? x : -INFINITY;
                    }
                    sr[c][i] = __float_as_uint(x);
                    mx = fmaxf(mx, x);
                }
            }
            const float m_new = fmaxf(m_ref, mx);
            // a row with nothing accumulated yet (O holds zeros) adopts the new maximum directly;
            // otherwise the reference only moves when the maximum grew by more than 2^8
            const bool rescale = m_ref != -INFINITY && m_new > m_ref + 8.f;
            if (m_ref == -INFINITY) m_ref = m_new;
            if (__any_sync(0xffffffffu, rescale)) {
                if (!wait_all(B_PVDONE, (j - 1) & 1, 41)) { ok = false; break; }
                tc_fence_after();
                const float alpha = rescale ? fast_exp2(m_ref - m_new) : 1.f;
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    uint32_t o[32];
                    tmem_ld32(lane_base + kColO + c * 32, o);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                    tmem_st32(lane_base + kColO + c * 32, o);
                }
                tmem_st_wait();
                if (rescale) { l *= alpha; m_ref = m_new; }
            }
            const float mref = m_ref == -INFINITY ? 0.f : m_ref;
            uint32_t pk[64];
            float rs = 0.f;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
#pragma unroll
                for (int i = 0; i < 32; i += 2) {
                    const float p0 = fast_exp2(__uint_as_float(sr[c][i]) - mref);
                    const float p1 = fast_exp2(__uint_as_float(sr[c][i + 1]) - mref);
                    rs += p0 + p1;
                    pk[c * 16 + i / 2] = pack_bf16x2(p0, p1);
                }
            }
            l += rs;
            // the P tile is free once PV_{j-1} has read it
            if (j >= 1 && !wait_all(B_PVDONE, (j - 1) & 1, 42)) { ok = false; break; }
#pragma unroll
            for (int c = 0; c < 16; ++c) {
                const uint32_t off = (uint32_t)(c >> 3) * kPanel + sw128_offset(row, (c & 7) * 8);
                *reinterpret_cast<uint4 *>(sp + off) = make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(bar(B_PFULL));
        }
        if (ok && wait_all(B_PVDONE, (ne - 1) & 1, 43)) {
            tc_fence_after();
            const float inv = l > 0.f ? 1.f / l : 0.f;
            __nv_bfloat16 *orow = prm.out + ((size_t)(t < prm.T ? t : 0) * prm.num_q_heads + h) * kD;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t o[32];
                tmem_ld32(lane_base + kColO + c * 32, o);
                tmem_ld_wait();
                if (t < prm.T) {
#pragma unroll
                    for (int i = 0; i < 32; i += 8) {
                        uint4 w;
                        w.x = pack_bf16x2(__uint_as_float(o[i]) * inv, __uint_as_float(o[i + 1]) * inv);
                        w.y = pack_bf16x2(__uint_as_float(o[i + 2]) * inv, __uint_as_float(o[i + 3]) * inv);
                        w.z = pack_bf16x2(__uint_as_float(o[i + 4]) * inv, __uint_as_float(o[i + 5]) * inv);
                        w.w = pack_bf16x2(__uint_as_float(o[i + 6]) * inv, __uint_as_float(o[i + 7]) * inv);
                        *reinterpret_cast<uint4 *>(orow + c * 32 + i) = w;
                    }
                }
            }
            if (t < prm.T) prm.lse[(size_t)t * prm.num_q_heads + h] = l > 0.f ? (m_ref + log2f(l)) * PADOC_LN2 : -INFINITY;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 5) {
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
    prm.scale_log2 = scale_log2;
    prm.out = (__nv_bfloat16 *)out;
    prm.lse = lse;
    prm.err = err;
    PADOC_CUDA_TRY(cudaFuncSetAttribute(prefill_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes));
    dim3 grid((unsigned)num_q_heads, (unsigned)nqt);
    prefill_tc_kernel<<<grid, 192, kSmemBytes, stream>>>(qmap, kmap, vmap, prm);
    return padoc_launch_status();
}
