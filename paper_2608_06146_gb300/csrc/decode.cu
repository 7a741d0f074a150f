// decode.cu -- C2/C4/C5: one decode step for every live stream over the paged KV cache
// (Algorithm 1's "decode o for all streams using the additive bias A_M", App. E.1), the split-K
// merge of partial softmax results, and the fp32 bring-up path.
//
// bf16 path. The planner cuts each page's shared stream into split-K pieces and each stream's
// private rows into pieces; a work item is one piece for one KV head. A shared item covers up to
// four streams of the page, so the piece's K/V is fetched from HBM once for all of them; every
// stream keeps its own column cutoff P + f_k. Each 16-token paged block is one TMA box per
// 64-column half (128-byte swizzle), staged through a 4-deep ring of 64-token stages.
//
// Warp-level math ("heads as the N dimension"): for one stream the 8 query heads of a KV head
// are the N = 8 columns of mma.m16n8k16, and the 16 tokens of a paged block are its M = 16 rows:
//     S^T[16 tok x 8 heads] = K[16 x 128] . Q^T[128 x 8]             (8 MMAs)
//     O^T[128 x 8 heads]   += V^T[128 x 16 tok] . P^T[16 tok x 8]    (8 MMAs)
// so no MMA lane is padding. The P^T operand is the score fragment transposed in registers with
// movmatrix; the online softmax runs per head over the token axis with shuffles.
#include <math.h>

#include <mutex>

#include "common.cuh"

namespace {

constexpr int kD = 128;          // head_dim of the bf16 path
constexpr int kGroup = 8;        // query heads per KV head of the bf16 path
constexpr int kBlk = 16;         // tokens per paged block
constexpr int kStageBlocks = 4;  // paged blocks per pipeline stage
constexpr int kStages = 4;       // pipeline depth
constexpr int kWarps = 4;
constexpr int kPanelBytes = kStageBlocks * kBlk * 128;   // [64 rows][64 cols] bf16
constexpr int kStageBytes = 4 * kPanelBytes;             // K lo, K hi, V lo, V hi
constexpr int kMergeStride = 132;                        // floats per head row of the merge area
constexpr int kMergeWarpFloats = kGroup * kMergeStride + 2 * kGroup;
constexpr size_t kDecodeSmem = 1024 + (size_t)kStages * kStageBytes + (size_t)kWarps * kMergeWarpFloats * 4 + 64;

struct DecodeParams {
    const int32_t *stream_page, *shared_len, *private_len, *slot_ptr;
    const padoc_item *items;
    const int32_t *page_table;
    const int32_t *stream_table;
    int32_t page_stride, stream_stride;
    int32_t num_blocks, num_kv_heads, num_q_heads;
    const __nv_bfloat16 *q;
    float *part_o, *part_lse;
    float scale_log2;
    int *err;
};

__global__ void __launch_bounds__(128, 1)
decode_mma_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                  const DecodeParams prm)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    float *merge = (float *)(smem + (size_t)kStages * kStageBytes);
    uint64_t *full_bar = (uint64_t *)(merge + kWarps * kMergeWarpFloats);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const padoc_item it = prm.items[blockIdx.x];
    const bool is_shared = it.kind == PADOC_ITEM_SHARED;
    const int nb = it.num_streams;
    const int wpb = nb == 1 ? 4 : (nb == 2 ? 2 : 1);   // warps per stream
    const int my_b = warp / wpb, phase = warp % wpb;
    const bool active = my_b < nb;
    const int g = it.kv_head;
    const int32_t *table = is_shared ? prm.page_table + (size_t)it.index * prm.page_stride
                                     : prm.stream_table + (size_t)it.index * prm.stream_stride;
    const int blk0 = it.tok_begin / kBlk;
    const int nblk = (it.tok_end - it.tok_begin + kBlk - 1) / kBlk;
    const int nstages = (nblk + kStageBlocks - 1) / kStageBlocks;

    if (tid == 0) {
        for (int i = 0; i < kStages; ++i) mbar_init(smem_u32(&full_bar[i]), 1);
        fence_barrier_init();
        tma_prefetch_desc(&kmap);
        tma_prefetch_desc(&vmap);
    }
    __syncthreads();

    auto issue = [&](int st) {
        const uint32_t base = smem_u32(smem + (size_t)(st % kStages) * kStageBytes);
        const uint32_t bar = smem_u32(&full_bar[st % kStages]);
        uint32_t bytes = 0;
        int32_t ids[kStageBlocks];
        for (int b = 0; b < kStageBlocks; ++b) {
            const int bi = st * kStageBlocks + b;
            ids[b] = -1;
            if (bi >= nblk) continue;
            const int32_t id = table[blk0 + bi];
            if (id < 0 || id >= prm.num_blocks) {
                padoc_record_error(prm.err, PADOC_DEVERR_BLOCK_ID, id);
                continue;
            }
            ids[b] = id;
            bytes += 4 * kBlk * 128;
        }
        mbar_arrive_expect_tx(bar, bytes);
        for (int b = 0; b < kStageBlocks; ++b) {
            if (ids[b] < 0) continue;
            const int32_t row = (ids[b] * prm.num_kv_heads + g) * kBlk;
            const uint32_t off = (uint32_t)b * (kBlk * 128);
            tma_load_2d(base + 0 * kPanelBytes + off, &kmap, 0, row, bar);
            tma_load_2d(base + 1 * kPanelBytes + off, &kmap, 64, row, bar);
            tma_load_2d(base + 2 * kPanelBytes + off, &vmap, 0, row, bar);
            tma_load_2d(base + 3 * kPanelBytes + off, &vmap, 64, row, bar);
        }
    };
    if (tid == 0)
        for (int st = 0; st < kStages && st < nstages; ++st) issue(st);

    // per-thread state: heads h0 = 2*(lane%4), h0+1 of this warp's stream
    const int s = it.first_stream + (active ? my_b : 0);
    int cutoff = 0;
    uint32_t qb[8][2];
    if (active) {
        cutoff = is_shared ? prm.shared_len[s] : prm.private_len[s];
        cutoff = min(cutoff, it.tok_end);
        const __nv_bfloat16 *qrow = prm.q + ((size_t)s * prm.num_q_heads + g * kGroup + (lane >> 2)) * kD;
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
            qb[ks][0] = *reinterpret_cast<const uint32_t *>(qrow + ks * 16 + (lane & 3) * 2);
            qb[ks][1] = *reinterpret_cast<const uint32_t *>(qrow + ks * 16 + 8 + (lane & 3) * 2);
        }
    }
    float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};
    float o[8][4];
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;

    int st = 0;
    bool aborted = false;
    for (; st < nstages; ++st) {
        const bool ok = mbar_wait_bounded(smem_u32(&full_bar[st % kStages]), (st / kStages) & 1, prm.err, 1);
        if (__syncthreads_or(!ok)) { aborted = true; break; }
        const uint32_t base = smem_u32(smem + (size_t)(st % kStages) * kStageBytes);
        if (active) {
            for (int j = 0; j < kStageBlocks; ++j) {
                const int bi = st * kStageBlocks + j;
                if (bi >= nblk || (bi % wpb) != phase) continue;
                const int tokbase = (blk0 + bi) * kBlk;
                if (tokbase >= cutoff) continue;
                // S^T = K . Q^T
                float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {
                    const uint32_t row = j * kBlk + (lane & 15);
                    const uint32_t col = (ks & 3) * 16 + (lane >> 4) * 8;
                    uint32_t a[4];
                    ldmatrix_x4(a, base + (ks >> 2) * kPanelBytes + sw128_offset(row, col));
                    mma_bf16_16816(acc, a, qb[ks][0], qb[ks][1]);
                }
                const int t0 = tokbase + (lane >> 2), t1 = t0 + 8;
                float sc[4];
                sc[0] = t0 < cutoff ? acc[0] * prm.scale_log2 : -INFINITY;
                sc[1] = t0 < cutoff ? acc[1] * prm.scale_log2 : -INFINITY;
                sc[2] = t1 < cutoff ? acc[2] * prm.scale_log2 : -INFINITY;
                sc[3] = t1 < cutoff ? acc[3] * prm.scale_log2 : -INFINITY;
                float mx0 = fmaxf(sc[0], sc[2]), mx1 = fmaxf(sc[1], sc[3]);
#pragma unroll
                for (int sh = 4; sh < 32; sh <<= 1) {
                    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, sh));
                    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, sh));
                }
                const float mn0 = fmaxf(m[0], mx0), mn1 = fmaxf(m[1], mx1);
                // a head whose columns are all masked so far keeps m = -inf and contributes 0
                const float al0 = mn0 == -INFINITY ? 1.f : fast_exp2(m[0] - mn0);
                const float al1 = mn1 == -INFINITY ? 1.f : fast_exp2(m[1] - mn1);
                const float p0 = mn0 == -INFINITY ? 0.f : fast_exp2(sc[0] - mn0);
                const float p1 = mn1 == -INFINITY ? 0.f : fast_exp2(sc[1] - mn1);
                const float p2 = mn0 == -INFINITY ? 0.f : fast_exp2(sc[2] - mn0);
                const float p3 = mn1 == -INFINITY ? 0.f : fast_exp2(sc[3] - mn1);
                m[0] = mn0; m[1] = mn1;
                l[0] = l[0] * al0 + p0 + p2;
                l[1] = l[1] * al1 + p1 + p3;
                const uint32_t b0 = movmatrix_trans(pack_bf16x2(p0, p1));
                const uint32_t b1 = movmatrix_trans(pack_bf16x2(p2, p3));
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {
                    o[mt][0] *= al0; o[mt][1] *= al1; o[mt][2] *= al0; o[mt][3] *= al1;
                    const int i = lane >> 3;
                    const uint32_t row = j * kBlk + (lane & 7) + (i >= 2 ? 8 : 0);
                    const uint32_t col = (mt & 3) * 16 + (i & 1) * 8;
                    uint32_t a[4];
                    ldmatrix_x4_trans(a, base + (2 + (mt >> 2)) * kPanelBytes + sw128_offset(row, col));
                    mma_bf16_16816(o[mt], a, b0, b1);
                }
            }
        }
        __syncthreads();
        if (tid == 0 && st + kStages < nstages) issue(st + kStages);
    }
    if (aborted) {
        // let the copies still in flight land before the CTA's shared memory is released
        if (tid == 0)
            for (int r = st + 1; r < nstages && r < st + kStages; ++r)
                mbar_wait_bounded(smem_u32(&full_bar[r % kStages]), (r / kStages) & 1, prm.err, 2);
        return;
    }

    // complete the row sums over the 8 token lanes of each head
#pragma unroll
    for (int sh = 4; sh < 32; sh <<= 1) {
        l[0] += __shfl_xor_sync(0xffffffffu, l[0], sh);
        l[1] += __shfl_xor_sync(0xffffffffu, l[1], sh);
    }
    float *mw = merge + warp * kMergeWarpFloats;   // [8 heads][kMergeStride] O^T, then m[8], l[8]
    if (active) {
        const int h0 = (lane & 3) * 2;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
            const int d0 = mt * 16 + (lane >> 2);
            mw[h0 * kMergeStride + d0] = o[mt][0];
            mw[(h0 + 1) * kMergeStride + d0] = o[mt][1];
            mw[h0 * kMergeStride + d0 + 8] = o[mt][2];
            mw[(h0 + 1) * kMergeStride + d0 + 8] = o[mt][3];
        }
        if (lane < 4) {
            mw[kGroup * kMergeStride + h0] = m[0];
            mw[kGroup * kMergeStride + h0 + 1] = m[1];
            mw[kGroup * kMergeStride + kGroup + h0] = l[0];
            mw[kGroup * kMergeStride + kGroup + h0 + 1] = l[1];
        }
    }
    __syncthreads();
    // merge the wpb warps of each stream and write this item's partial results
    for (int idx = tid; idx < nb * kGroup * kD; idx += blockDim.x) {
        const int b = idx / (kGroup * kD), hl = (idx / kD) % kGroup, dd = idx % kD;
        float mstar = -INFINITY;
        for (int w = 0; w < wpb; ++w)
            mstar = fmaxf(mstar, merge[(b * wpb + w) * kMergeWarpFloats + kGroup * kMergeStride + hl]);
        float lsum = 0.f, osum = 0.f;
        if (mstar != -INFINITY) {
            for (int w = 0; w < wpb; ++w) {
                const float *mwp = merge + (b * wpb + w) * kMergeWarpFloats;
                const float f = exp2f(mwp[kGroup * kMergeStride + hl] - mstar);
                lsum += f * mwp[kGroup * kMergeStride + kGroup + hl];
                osum += f * mwp[hl * kMergeStride + dd];
            }
        }
        const int sidx = it.first_stream + b;
        const int slot = prm.slot_ptr[sidx] + it.slot;
        const int h = g * kGroup + hl;
        const size_t row = (size_t)slot * prm.num_q_heads + h;
        const bool empty = !(lsum > 0.f);
        prm.part_o[row * kD + dd] = empty ? 0.f : osum / lsum;
        if (dd == 0) prm.part_lse[row] = empty ? -INFINITY : (mstar + log2f(lsum)) * PADOC_LN2;
    }
}

// ------------------------------------------------------------------------------------------------
// Split-K merge (C4): one warp per output row, 4 consecutive dims per lane.
// ------------------------------------------------------------------------------------------------
struct RaggedSlots {   // decode: row = s * Hq + h, slots [slot_ptr[s], slot_ptr[s+1])
    const int32_t *slot_ptr;
    int32_t hq;
    __device__ int count(int64_t row) const { return slot_ptr[row / hq + 1] - slot_ptr[row / hq]; }
    __device__ int64_t part_row(int64_t row, int i) const { return (int64_t)(slot_ptr[row / hq] + i) * hq + row % hq; }
};
struct UniformSlots {  // public combine: part_row = split * rows + row
    int32_t splits;
    int64_t rows;
    __device__ int count(int64_t) const { return splits; }
    __device__ int64_t part_row(int64_t row, int i) const { return (int64_t)i * rows + row; }
};

template <class Slots, class OutT>
__global__ void __launch_bounds__(128) combine_kernel(Slots sl, const float *__restrict__ part_o,
                                                      const float *__restrict__ part_lse, int64_t rows, int d,
                                                      OutT *__restrict__ out, float *__restrict__ lse_out)
{
    const int64_t row = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= rows) return;
    const int n = sl.count(row);
    float mx = -INFINITY;
    for (int i = lane; i < n; i += 32) mx = fmaxf(mx, part_lse[sl.part_row(row, i)]);
#pragma unroll
    for (int sh = 16; sh > 0; sh >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, sh));
    float sum = 0.f;
    if (mx != -INFINITY)
        for (int i = lane; i < n; i += 32) sum += expf(part_lse[sl.part_row(row, i)] - mx);
#pragma unroll
    for (int sh = 16; sh > 0; sh >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, sh);
    const float tot = mx == -INFINITY ? -INFINITY : mx + logf(sum);
    for (int c0 = lane * 4; c0 < d; c0 += 128) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        if (tot != -INFINITY) {
            for (int i = 0; i < n; ++i) {
                const int64_t pr = sl.part_row(row, i);
                const float w = expf(part_lse[pr] - tot);
                if (w == 0.f) continue;
                const float4 v = *reinterpret_cast<const float4 *>(part_o + pr * d + c0);
                acc.x += w * v.x; acc.y += w * v.y; acc.z += w * v.z; acc.w += w * v.w;
            }
        }
        if constexpr (sizeof(OutT) == 2) {
            uint2 pk;
            pk.x = pack_bf16x2(acc.x, acc.y);
            pk.y = pack_bf16x2(acc.z, acc.w);
            *reinterpret_cast<uint2 *>(reinterpret_cast<__nv_bfloat16 *>(out) + row * d + c0) = pk;
        } else {
            *reinterpret_cast<float4 *>(reinterpret_cast<float *>(out) + row * d + c0) = acc;
        }
    }
    if (lane == 0 && lse_out) lse_out[row] = tot;
}

// ------------------------------------------------------------------------------------------------
// fp32 bring-up path: one warp per (stream, query head), keys visited in order, online softmax.
// ------------------------------------------------------------------------------------------------
template <int D>
__global__ void __launch_bounds__(128) decode_f32_kernel(const float *__restrict__ k_pool, const float *__restrict__ v_pool,
                                                         int32_t num_blocks, int32_t hkv, const int32_t *stream_page,
                                                         const int32_t *shared_len, const int32_t *private_len,
                                                         const int32_t *page_table, int32_t page_stride,
                                                         const int32_t *stream_table, int32_t stream_stride,
                                                         const float *__restrict__ q, int32_t num_streams, int32_t hq,
                                                         float scale_log2, float *__restrict__ out,
                                                         float *__restrict__ lse, int *err)
{
    constexpr int E = D / 32;
    const int64_t row = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= (int64_t)num_streams * hq) return;
    const int s = (int)(row / hq), h = (int)(row % hq), g = h / (hq / hkv);
    float qv[E], ov[E];
#pragma unroll
    for (int e = 0; e < E; ++e) { qv[e] = q[row * D + lane + 32 * e]; ov[e] = 0.f; }
    float m = -INFINITY, l = 0.f;
    for (int part = 0; part < 2; ++part) {
        const int n = part == 0 ? shared_len[s] : private_len[s];
        const int32_t *table = part == 0 ? page_table + (size_t)stream_page[s] * page_stride
                                         : stream_table + (size_t)s * stream_stride;
        for (int t = 0; t < n; ++t) {
            const int32_t id = table[t / 16];
            if (id < 0 || id >= num_blocks) {
                if (lane == 0) padoc_record_error(err, PADOC_DEVERR_BLOCK_ID, id);
                continue;
            }
            const size_t kr = (((size_t)id * hkv + g) * 16 + (t % 16)) * D;
            float dot = 0.f;
#pragma unroll
            for (int e = 0; e < E; ++e) dot = fmaf(qv[e], k_pool[kr + lane + 32 * e], dot);
#pragma unroll
            for (int sh = 16; sh > 0; sh >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, sh);
            const float sc = dot * scale_log2;
            const float mn = fmaxf(m, sc);
            const float al = exp2f(m - mn), p = exp2f(sc - mn);
            l = l * al + p;
#pragma unroll
            for (int e = 0; e < E; ++e) ov[e] = fmaf(p, v_pool[kr + lane + 32 * e], ov[e] * al);
            m = mn;
        }
    }
    const bool empty = !(l > 0.f);
#pragma unroll
    for (int e = 0; e < E; ++e) out[row * D + lane + 32 * e] = empty ? 0.f : ov[e] / l;
    if (lane == 0) lse[row] = empty ? -INFINITY : (m + log2f(l)) * PADOC_LN2;
}

}  // namespace

// ------------------------------------------------------------------------------------------------
// Host entry points
// ------------------------------------------------------------------------------------------------

extern "C" padoc_status padoc_branch_decode_attn(const padoc_kv_pool *pool, const padoc_decode_plan *info,
                                                 const int32_t *plan_dev, const int32_t *page_block_table,
                                                 int32_t page_table_stride, const int32_t *stream_block_table,
                                                 int32_t stream_table_stride, const void *q, float scale, void *out,
                                                 float *lse, void *workspace, size_t workspace_bytes,
                                                 padoc_stream_t stream)
{
    if (!pool || !info || !plan_dev || !q || !out || !lse) return PADOC_ERR_INVALID_ARGUMENT;
    const padoc_decode_config &cfg = info->cfg;
    if (pool->block_size != cfg.block_size || pool->num_kv_heads != cfg.num_kv_heads || pool->head_dim != cfg.head_dim)
        return PADOC_ERR_INVALID_ARGUMENT;
    if (!pool->k_pool || !pool->v_pool || pool->num_blocks < 1) return PADOC_ERR_INVALID_ARGUMENT;
    if (!(scale > 0.f) || !isfinite(scale)) return PADOC_ERR_INVALID_ARGUMENT;
    if (info->num_pages > 0 && (!page_block_table || page_table_stride < info->max_page_blocks))
        return PADOC_ERR_INVALID_ARGUMENT;
    if (info->num_streams > 0 && (!stream_block_table || stream_table_stride < info->max_stream_blocks))
        return PADOC_ERR_INVALID_ARGUMENT;
    if (info->num_streams == 0) return PADOC_OK;
    if ((((uintptr_t)pool->k_pool) | ((uintptr_t)pool->v_pool) | ((uintptr_t)q) | ((uintptr_t)out)) & 15)
        return PADOC_ERR_INVALID_ARGUMENT;
    const int32_t *plan = plan_dev;
    int *err = padoc_device_error_word();
    if (!err) return PADOC_ERR_CUDA;
    cudaStream_t cs = (cudaStream_t)stream;

    if (pool->dtype == PADOC_DTYPE_F32) {
        if (cfg.head_dim != 64 && cfg.head_dim != 128) return PADOC_ERR_UNSUPPORTED;
        const int64_t rows = (int64_t)info->num_streams * cfg.num_q_heads;
        const unsigned grid = (unsigned)((rows + 3) / 4);
        const float sl2 = scale * PADOC_LOG2E;
#define PADOC_F32_DECODE(DIM)                                                                                    \
    decode_f32_kernel<DIM><<<grid, 128, 0, cs>>>(                                                               \
        (const float *)pool->k_pool, (const float *)pool->v_pool, pool->num_blocks, cfg.num_kv_heads,           \
        plan + info->off_stream_page, plan + info->off_shared_len, plan + info->off_private_len, page_block_table, \
        page_table_stride, stream_block_table, stream_table_stride, (const float *)q, info->num_streams,         \
        cfg.num_q_heads, sl2, (float *)out, lse, err)
        if (cfg.head_dim == 64) PADOC_F32_DECODE(64); else PADOC_F32_DECODE(128);
#undef PADOC_F32_DECODE
        return padoc_launch_status();
    }
    if (pool->dtype != PADOC_DTYPE_BF16) return PADOC_ERR_UNSUPPORTED;
    if (cfg.head_dim != kD || cfg.num_q_heads != kGroup * cfg.num_kv_heads || cfg.block_size != kBlk)
        return PADOC_ERR_UNSUPPORTED;
    size_t need = 0;
    padoc_decode_workspace_size(info, &need);
    if (!workspace || workspace_bytes < need) return PADOC_ERR_WORKSPACE_TOO_SMALL;
    if (((uintptr_t)workspace) & 255) return PADOC_ERR_INVALID_ARGUMENT;

    const uint64_t rows = (uint64_t)pool->num_blocks * cfg.num_kv_heads * kBlk;
    CUtensorMap kmap, vmap;
    if (!padoc_make_tmap_bf16(&kmap, pool->k_pool, kD, rows, kD * 2, 64, kBlk) ||
        !padoc_make_tmap_bf16(&vmap, pool->v_pool, kD, rows, kD * 2, 64, kBlk))
        return PADOC_ERR_CUDA;

    DecodeParams prm;
    prm.stream_page = plan + info->off_stream_page;
    prm.shared_len = plan + info->off_shared_len;
    prm.private_len = plan + info->off_private_len;
    prm.slot_ptr = plan + info->off_slot_ptr;
    prm.items = reinterpret_cast<const padoc_item *>(plan + info->off_items);
    prm.page_table = page_block_table;
    prm.stream_table = stream_block_table;
    prm.page_stride = page_table_stride;
    prm.stream_stride = stream_table_stride;
    prm.num_blocks = pool->num_blocks;
    prm.num_kv_heads = cfg.num_kv_heads;
    prm.num_q_heads = cfg.num_q_heads;
    prm.q = (const __nv_bfloat16 *)q;
    prm.part_o = (float *)workspace;
    prm.part_lse = (float *)((uint8_t *)workspace + padoc_align256((size_t)info->num_slots * cfg.num_q_heads * kD * 4));
    prm.scale_log2 = scale * PADOC_LOG2E;
    prm.err = err;

    static bool attr_set = false;   // per process; the attribute is per function
    if (!attr_set) {
        PADOC_CUDA_TRY(cudaFuncSetAttribute(decode_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kDecodeSmem));
        attr_set = true;
    }
    if (info->num_items > 0) {
        decode_mma_kernel<<<info->num_items, 128, kDecodeSmem, cs>>>(kmap, vmap, prm);
        padoc_status st = padoc_launch_status();
        if (st != PADOC_OK) return st;
    }
    const int64_t out_rows = (int64_t)info->num_streams * cfg.num_q_heads;
    RaggedSlots sl{prm.slot_ptr, cfg.num_q_heads};
    combine_kernel<RaggedSlots, __nv_bfloat16><<<(unsigned)((out_rows + 3) / 4), 128, 0, cs>>>(
        sl, prm.part_o, prm.part_lse, out_rows, kD, (__nv_bfloat16 *)out, lse);
    return padoc_launch_status();
}

extern "C" padoc_status padoc_splitk_combine(const float *part_o, const float *part_lse, int32_t num_splits,
                                             int64_t rows, int32_t head_dim, padoc_dtype out_dtype, void *out,
                                             float *lse, padoc_stream_t stream)
{
    if (num_splits < 0 || rows < 0 || head_dim < 4 || head_dim > 256 || head_dim % 4 != 0) return PADOC_ERR_INVALID_ARGUMENT;
    if (rows == 0) return PADOC_OK;
    if (!out || (num_splits > 0 && (!part_o || !part_lse))) return PADOC_ERR_INVALID_ARGUMENT;
    if ((((uintptr_t)part_o) & 15) || (((uintptr_t)out) & 7)) return PADOC_ERR_INVALID_ARGUMENT;
    UniformSlots sl{num_splits, rows};
    const unsigned grid = (unsigned)((rows + 3) / 4);
    cudaStream_t cs = (cudaStream_t)stream;
    if (out_dtype == PADOC_DTYPE_BF16)
        combine_kernel<UniformSlots, __nv_bfloat16><<<grid, 128, 0, cs>>>(sl, part_o, part_lse, rows, head_dim,
                                                                         (__nv_bfloat16 *)out, lse);
    else if (out_dtype == PADOC_DTYPE_F32)
        combine_kernel<UniformSlots, float><<<grid, 128, 0, cs>>>(sl, part_o, part_lse, rows, head_dim, (float *)out, lse);
    else
        return PADOC_ERR_INVALID_ARGUMENT;
    return padoc_launch_status();
}

// ------------------------------------------------------------------------------------------------
// Decode without caller-provided workspace.
//
// Some callers cannot allocate device memory: a plugin inside a host framework that owns all device
// memory and hands its plugins no allocator, or a latency-critical decode loop where a cudaMalloc
// (which may synchronize the device) is not acceptable. For them the split-K partials live in a
// fixed array that every device loading this library holds until the process exits.
// ------------------------------------------------------------------------------------------------
namespace {

__device__ __align__(256) uint8_t g_static_workspace[PADOC_STATIC_WORKSPACE_BYTES];

constexpr int kMaxStaticDevices = 64;
void *g_static_ws_ptr[kMaxStaticDevices] = {nullptr};
std::mutex g_static_ws_mu;

// Device address of this device's copy of the array. Host code must not pass the symbol itself to a
// kernel: on the host it names a host-side stand-in, not device memory.
void *static_workspace_address()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxStaticDevices) return nullptr;
    std::lock_guard<std::mutex> lk(g_static_ws_mu);
    if (!g_static_ws_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_workspace) != cudaSuccess) return nullptr;
        g_static_ws_ptr[dev] = p;
    }
    return g_static_ws_ptr[dev];
}

}  // namespace

extern "C" padoc_status padoc_branch_decode_attn_noalloc(const padoc_kv_pool *pool, const padoc_decode_plan *info,
                                                         const int32_t *plan_dev, const int32_t *page_block_table,
                                                         int32_t page_table_stride, const int32_t *stream_block_table,
                                                         int32_t stream_table_stride, const void *q, float scale,
                                                         void *out, float *lse, padoc_stream_t stream)
{
    if (!info) return PADOC_ERR_INVALID_ARGUMENT;
    size_t need = 0;
    padoc_status st = padoc_decode_workspace_size(info, &need);
    if (st != PADOC_OK) return st;
    if (need > (size_t)PADOC_STATIC_WORKSPACE_BYTES) return PADOC_ERR_WORKSPACE_TOO_SMALL;
    void *ws = static_workspace_address();
    if (!ws) return PADOC_ERR_CUDA;
    return padoc_branch_decode_attn(pool, info, plan_dev, page_block_table, page_table_stride, stream_block_table,
                                    stream_table_stride, q, scale, out, lse, ws, (size_t)PADOC_STATIC_WORKSPACE_BYTES,
                                    stream);
}
