// decode_tc.cu -- C2 on the 5th-generation tensor cores: the shared-stream part of one decode step.
//
// For a page whose branches x query heads (of one KV head) fill dense M = 128 tiles, a work item
// covers a split-K piece [tok_begin, tok_end) of the page's shared stream (prefix + layout, stored
// once in the paged KV cache) for up to 32 of its streams: two M-tiles of 16 streams x 8 query
// heads. Each K/V tile of 128 tokens is fetched from HBM once and multiplied against every
// stream's queries; row (stream b, head h) sees the columns before its own cutoff P + f_k
// (Algorithm 1's mask row restricted to the shared stream). The item writes one partial
// (normalized O, natural-log LSE) per (stream, head) into its split-K slot; the merge kernel joins
// the shared-stream and private-history partials.
//
// The CTA layout follows the packed-prefill kernel: warps 0-3 / 4-7 run the softmax of M-tile 0 / 1
// (thread t owns row t), warp 8 is the TMA producer (the item's queries as one 4-D box per panel;
// the item's block rows looked up once; then lanes 0-7 each fetch one 16-token paged block of K and
// of V per tile, two 64-column boxes each; blocks past the piece or with an out-of-range id are
// fetched from an out-of-range coordinate, which fills zeros), warp 9 allocates TMEM and issues the
// MMAs as a converged warp. A stage's K is released when the tile's last QK^T completes and its V
// when the last PV completes. TMEM: S_i / P_i at columns 128i, O_i at 256 + 128i.
#include <math.h>

#include "common.cuh"
#include "tc.cuh"

namespace {

constexpr int kD = 128;
constexpr int kGroup = 8;        // query heads per KV head
constexpr int kBlk = 16;         // tokens per paged block
constexpr int kKT = 128;         // tokens per K/V tile
constexpr int kPanel = 128 * 128;
constexpr int kTile = 2 * kPanel;
constexpr int kStages = 2;
constexpr uint32_t kTmemCols = 512;
constexpr int kThreads = 320;

enum {
    B_Q = 0,
    B_KFULL = 1,     // [stage]
    B_VFULL = 3,     // [stage]
    B_KEMPTY = 5,    // [stage]: the last QK^T of the tile has completed
    B_VEMPTY = 7,    // [stage]: the last PV of the tile has completed
    B_SFULL = 9,     // [m-tile]
    B_PFULL = 11,    // [m-tile], 128 arrivals
    B_PVDONE = 13,   // [m-tile]
    B_FINAL = 15,
    B_COUNT = 16
};

constexpr int kMaxItemBlocks = PADOC_TC_MAX_ITEM_TOKENS / kBlk;   // block rows an item looks up once
constexpr size_t kSmemBytes = 1024 + (size_t)kTile * (2 + 2 * kStages) + B_COUNT * 8 + 64 + kMaxItemBlocks * 4;

struct TcDecodeParams {
    const int32_t *shared_len, *slot_ptr;
    const padoc_item *items;
    const int32_t *page_table;
    int32_t page_stride;
    int32_t num_blocks, num_kv_heads, num_q_heads;
    int32_t pool_rows;           // num_blocks * num_kv_heads * 16: first out-of-range row
    const __nv_bfloat16 *q;
    float *part_o, *part_lse;
    float scale_log2;
    int *err;
};

__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, int *err, int site, volatile int *abort_flag)
{
    if (*abort_flag) return false;
    if (mbar_wait_bounded(bar, parity, err, site)) return true;
    *abort_flag = 1;
    return false;
}

template <int MT>
__device__ __forceinline__ void decode_tc_body(const CUtensorMap *kmap, const CUtensorMap *vmap, const CUtensorMap *qmap,
                                               const TcDecodeParams &prm, const padoc_item &it, uint8_t *smem,
                                               uint64_t *bars, int32_t *block_rows, uint32_t tmem,
                                               volatile int *abort_flag)
{
    uint8_t *sq = smem;
    uint8_t *sk = sq + 2 * kTile;
    uint8_t *sv = sk + kStages * kTile;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = it.kv_head;
    const int tb = it.tok_begin, te = it.tok_end;
    const int ne = (te - tb + kKT - 1) / kKT;   // K/V tiles of this piece
    auto bar = [&](int i) { return smem_u32(&bars[i]); };

    if (warp == 8) {
        // ---------------------------------------------------------------- TMA producer (whole warp)
        // queries first: one 4-D box per 64-column panel gathers 16 streams x 8 heads of KV head g
        if (lane == 0 && ne > 0) {
            mbar_arrive_expect_tx(bar(B_Q), MT * kTile);
#pragma unroll
            for (int i = 0; i < MT; ++i) {
                tma_load_4d(smem_u32(sq + i * kTile), qmap, 0, 0, g, it.first_stream + 16 * i, bar(B_Q));
                tma_load_4d(smem_u32(sq + i * kTile) + kPanel, qmap, 64, 0, g, it.first_stream + 16 * i, bar(B_Q));
            }
        }
        // the item's block rows, looked up once (out-of-range ids and blocks past the piece read
        // from an out-of-range row, which fills zeros)
        const int32_t *table = prm.page_table + (size_t)it.index * prm.page_stride;
        const int nblk = ne * (kKT / kBlk);
        auto lookup = [&](int bi) {
            const int tok0 = tb + bi * kBlk;
            int32_t row = prm.pool_rows;
            if (tok0 < te) {
                const int32_t id = table[tok0 / kBlk];
                if (id >= 0 && id < prm.num_blocks) row = (id * prm.num_kv_heads + g) * kBlk;
                else padoc_record_error(prm.err, PADOC_DEVERR_BLOCK_ID, id);
            }
            block_rows[bi] = row;
        };
        // the first tile's rows first, so its loads start before the remaining lookups
        if (lane < kKT / kBlk && lane < nblk) lookup(lane);
        __syncwarp();
        int issued = 0;
        for (int j = 0; j < ne; ++j) {
            if (j == 1) {
                for (int bi = kKT / kBlk + lane; bi < nblk; bi += 32) lookup(bi);
                __syncwarp();
            }
            const int s = j & 1;
            const uint32_t off = (uint32_t)lane * (kBlk * 128);
            const int32_t row = lane < kKT / kBlk ? block_rows[j * (kKT / kBlk) + lane] : 0;
            bool ok = true;
            if (j >= 2) ok = wait_or_abort(bar(B_KEMPTY + s), ((j - 2) >> 1) & 1, prm.err, 50, abort_flag);
            if (!__all_sync(0xffffffffu, ok)) break;
            if (lane == 0) mbar_arrive_expect_tx(bar(B_KFULL + s), kTile);
            __syncwarp();
            if (lane < kKT / kBlk) {
                const uint32_t kb = smem_u32(sk + s * kTile) + off;
                tma_load_2d(kb, kmap, 0, row, bar(B_KFULL + s));
                tma_load_2d(kb + kPanel, kmap, 64, row, bar(B_KFULL + s));
            }
            if (j >= 2) ok = wait_or_abort(bar(B_VEMPTY + s), ((j - 2) >> 1) & 1, prm.err, 53, abort_flag);
            if (!__all_sync(0xffffffffu, ok)) break;
            if (lane == 0) mbar_arrive_expect_tx(bar(B_VFULL + s), kTile);
            __syncwarp();
            if (lane < kKT / kBlk) {
                const uint32_t vb = smem_u32(sv + s * kTile) + off;
                tma_load_2d(vb, vmap, 0, row, bar(B_VFULL + s));
                tma_load_2d(vb + kPanel, vmap, 64, row, bar(B_VFULL + s));
            }
            issued = j + 1;
        }
        // copies still in flight must land before the CTA's shared memory is released
        if (lane == 0) {
            if (ne > 0) mbar_wait_bounded(bar(B_Q), 0, prm.err, 54);
            for (int j = (issued > 2 ? issued - 2 : 0); j < issued; ++j) {
                mbar_wait_bounded(bar(B_KFULL + (j & 1)), (j >> 1) & 1, prm.err, 51);
                mbar_wait_bounded(bar(B_VFULL + (j & 1)), (j >> 1) & 1, prm.err, 52);
            }
        }
    } else if (warp == 9) {
        // ---------------------------------------------------------------- MMA issuer (whole warp)
        constexpr uint32_t idS = umma_idesc_bf16(128, kKT, false);
        constexpr uint32_t idPV = umma_idesc_bf16(128, kD, true);
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
        bool ok = ne > 0 && wait_w(B_Q, 0, 60) && wait_w(B_KFULL, 0, 61);
        if (ok) {
            tc_fence_after();
#pragma unroll
            for (int i = 0; i < MT; ++i) issue_s(i, 0);
            umma_commit_warp(bar(B_KEMPTY));
        }
        for (int j = 0; ok && j < ne; ++j) {
            const int s = j & 1, sn = (j + 1) & 1;
#pragma unroll
            for (int i = 0; i < MT; ++i) {
                if (!wait_w(B_PFULL + i, j & 1, 62)) { ok = false; break; }
                if (i == 0 && !wait_w(B_VFULL + s, (j >> 1) & 1, 63)) { ok = false; break; }
                tc_fence_after();
                const uint64_t db = s ? dv1 : dv0;
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)
                    umma_bf16_ts_warp(tmem + 256 + 128 * i, tmem + 128 * i + kk * 8, db + kk * (2048 >> 4), idPV,
                                      (j > 0 || kk > 0));
                umma_commit_warp(bar(B_PVDONE + i));
                if (i == MT - 1) umma_commit_warp(bar(B_VEMPTY + s));
                if (j + 1 < ne) {
                    if (i == 0 && !wait_w(B_KFULL + sn, ((j + 1) >> 1) & 1, 64)) { ok = false; break; }
                    tc_fence_after();
                    issue_s(i, sn);
                    if (i == MT - 1) umma_commit_warp(bar(B_KEMPTY + sn));
                }
            }
        }
        // every MMA issued above must complete before TMEM is released
        umma_commit_warp(bar(B_FINAL));
        mbar_wait_bounded(bar(B_FINAL), 0, prm.err, 65);
    } else if (warp / 4 < MT) {
        // ---------------------------------------------------------------- queries, softmax, epilogue
        const int mi = warp / 4;                    // M-tile
        const int row = tid & 127;
        const int b = mi * 16 + row / kGroup, hl = row % kGroup;
        const bool valid = b < it.num_streams;
        const int s = it.first_stream + (valid ? b : 0);
        const int h = g * kGroup + hl;
        const int cutoff = valid ? min(prm.shared_len[s], te) : tb;   // visible tokens end here
        const uint32_t lanes = (uint32_t)((warp & 3) * 32) << 16;
        const uint32_t tS = tmem + lanes + 128 * mi, tO = tmem + lanes + 256 + 128 * mi;
        const float c = prm.scale_log2;
        auto wait_all = [&](int bb, uint32_t parity, int site) {
            const bool r = wait_or_abort(bar(bb), parity, prm.err, site, abort_flag);
            return __all_sync(0xffffffffu, r);
        };
        float m_ref = -INFINITY, l = 0.f;
        bool ok = ne > 0;
        for (int j = 0; ok && j < ne; ++j) {
            const int w = min(max(cutoff - (tb + j * kKT), 0), kKT);   // visible columns [0, w)
            const bool full = __all_sync(0xffffffffu, w == kKT);
            if (!wait_all(B_SFULL + mi, j & 1, 70)) { ok = false; break; }
            tc_fence_after();
            float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
            for (int q = 0; q < 4; q += 2) {
                uint32_t sr[2][32];
                tmem_ld32(tS + q * 32, sr[0]);
                tmem_ld32(tS + q * 32 + 32, sr[1]);
                tmem_ld_wait();
                if (!full) {
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
                        const uint32_t vis = interval_bits(0, w, (q + u) * 32);
#pragma unroll
                        for (int i = 0; i < 32; ++i) sr[u][i] = (vis >> i) & 1u ? sr[u][i] : 0xff800000u;
                        tmem_st32(tS + (q + u) * 32, sr[u]);
                    }
                }
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
            if (!full) tmem_st_wait();
            const float mx = fmaxf(fmax3f(mx4[0], mx4[1], mx4[2]), mx4[3]);
            const float m_new = fmaxf(m_ref, mx);
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
            mbar_arrive(bar(B_PFULL + mi));
        }
        // partial result of this piece: O / l (fp32) and its natural-log LSE
        const bool have = ne == 0 || (ok && wait_all(B_PVDONE + mi, (ne - 1) & 1, 71));
        if (have) {
            tc_fence_after();
            const bool empty = !(l > 0.f);
            const float inv = empty ? 0.f : 1.f / l;
            const size_t prow = (size_t)(prm.slot_ptr[s] + it.slot) * prm.num_q_heads + h;
            float *dst = prm.part_o + prow * kD;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                uint32_t o[32];
                if (ne > 0) {
                    tmem_ld32(tO + q * 32, o);
                    tmem_ld_wait();
                }
                if (valid) {
#pragma unroll
                    for (int i = 0; i < 32; i += 4)
                        *reinterpret_cast<float4 *>(dst + q * 32 + i) =
                            empty ? make_float4(0.f, 0.f, 0.f, 0.f)
                                  : make_float4(__uint_as_float(o[i]) * inv, __uint_as_float(o[i + 1]) * inv,
                                                __uint_as_float(o[i + 2]) * inv, __uint_as_float(o[i + 3]) * inv);
                }
            }
            if (valid) prm.part_lse[prow] = empty ? -INFINITY : (m_ref * c + log2f(l)) * PADOC_LN2;
        }
    }
}

__global__ void __launch_bounds__(kThreads, 1)
decode_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                 const __grid_constant__ CUtensorMap qmap, const TcDecodeParams prm)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t *bars = (uint64_t *)(smem + (size_t)kTile * (2 + 2 * kStages));
    uint32_t *tmem_slot = (uint32_t *)(bars + B_COUNT);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    int32_t *block_rows = (int32_t *)(tmem_slot + 16);
    const int tid = threadIdx.x, warp = tid >> 5;
    // the warp kernel that follows reads nothing this grid writes before its final wait, so it may
    // start filling SMs as soon as every CTA of this grid is resident
    pdl_launch_dependents();
    const padoc_item it = prm.items[blockIdx.x];
    const int mt = it.num_streams > 16 ? 2 : 1;

    if (tid == 0) {
        for (int i = 0; i < B_COUNT; ++i) {
            uint32_t cnt = 1;
            if (i == B_PFULL || i == B_PFULL + 1) cnt = 128;
            mbar_init(smem_u32(&bars[i]), cnt);
        }
        *abort_flag = 0;
        fence_barrier_init();
        tma_prefetch_desc(&kmap);
        tma_prefetch_desc(&vmap);
        tma_prefetch_desc(&qmap);
    }
    if (warp == 9) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    if (mt == 2) decode_tc_body<2>(&kmap, &vmap, &qmap, prm, it, smem, bars, block_rows, tmem, abort_flag);
    else decode_tc_body<1>(&kmap, &vmap, &qmap, prm, it, smem, bars, block_rows, tmem, abort_flag);
    tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

padoc_status padoc_launch_decode_tc(const CUtensorMap *kmap, const CUtensorMap *vmap, const CUtensorMap *qmap, const int32_t *plan,
                                    const padoc_decode_plan *info, const int32_t *page_table, int32_t page_stride,
                                    int32_t num_blocks, const void *q, float *part_o, float *part_lse, float scale_log2,
                                    int *err, cudaStream_t stream)
{
    if (info->num_tc_items == 0) return PADOC_OK;
    TcDecodeParams prm;
    prm.shared_len = plan + info->off_shared_len;
    prm.slot_ptr = plan + info->off_slot_ptr;
    prm.items = reinterpret_cast<const padoc_item *>(plan + info->off_items);
    prm.page_table = page_table;
    prm.page_stride = page_stride;
    prm.num_blocks = num_blocks;
    prm.num_kv_heads = info->cfg.num_kv_heads;
    prm.num_q_heads = info->cfg.num_q_heads;
    prm.pool_rows = num_blocks * info->cfg.num_kv_heads * kBlk;
    prm.q = (const __nv_bfloat16 *)q;
    prm.part_o = part_o;
    prm.part_lse = part_lse;
    prm.scale_log2 = scale_log2;
    prm.err = err;
    PADOC_CUDA_TRY(cudaFuncSetAttribute(decode_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes));
    decode_tc_kernel<<<info->num_tc_items, kThreads, kSmemBytes, stream>>>(*kmap, *vmap, *qmap, prm);
    return padoc_launch_status();
}
