// decode_warp.cuh -- C2/C5: the warp path of one decode step, shared by the stand-alone warp
// kernel (decode.cu) and the fused decode grid, whose CTAs run it after their tensor-core pieces
// (decode_tc.cu).
//
// Every warp owns one work item and runs on its own: a 3-deep ring of 16-token
// paged blocks fetched with cp.async (each lane copies 16 of the block's 512 16-byte chunks into
// a 128-byte-swizzled [16][64] panel per half of K and V), one cp.async group per block, so no
// warp ever waits for another. cp.async rather than TMA: a 16-token block is only four 2 KB
// boxes, and an SM issues a TMA box only every ~70 cycles. The math puts the 8 query heads of a KV head
// in the N = 8 columns of mma.m16n8k16 and the 16 tokens of a block in its M = 16 rows:
//     S^T[16 tok x 8 heads] = K[16 x 128] . Q^T[128 x 8]             (8 MMAs)
//     O^T[128 x 8 heads]   += V^T[128 x 16 tok] . P^T[16 tok x 8]    (8 MMAs)
// so no MMA lane is padding. The P^T operand is the score fragment transposed in registers with
// movmatrix; the online softmax runs per head over the token axis with shuffles.
#pragma once

#include <math.h>

#include "common.cuh"

namespace padoc_warp {

constexpr int kD = 128;          // head_dim of the bf16 path
constexpr int kGroup = 8;        // query heads per KV head of the bf16 path
constexpr int kBlk = 16;         // tokens per paged block
constexpr int kWarps = PADOC_WARP_KERNEL_WARPS;   // independent warps per CTA
constexpr int kWStages = 3;            // paged blocks in flight per warp
constexpr int kBoxBytes = kBlk * 128;  // one 16-row x 64-column box
constexpr int kWStageBytes = 4 * kBoxBytes;   // K lo, K hi, V lo, V hi
constexpr int kWarpRing = kWStages * kWStageBytes;
// E4M3 pool: a stage holds a block's K and V codes ([16 rows][128 bytes] each, 16-byte chunks
// swizzled by row) and its two scales; each warp expands the block it works on into one bf16
// buffer laid out as a bf16 stage, which the MMAs read.
constexpr int kE8Rows = kBlk * 128;                  // 2 KB of codes per tensor
constexpr int kE8StageBytes = 2 * kE8Rows + 128;     // K codes, V codes, scales (k, v)
constexpr int kE8WarpBytes = kWStages * kE8StageBytes + kWStageBytes;
// shared memory of the kWarps warps' rings, from a 1024-byte-aligned base
constexpr size_t kRingBytes = (size_t)kWarps * kWarpRing;
constexpr size_t kRingBytesE4M3 = (size_t)kWarps * kE8WarpBytes;
constexpr float kTwo112 = 5.192296858534828e33f;     // 2^112: the bf16 expansion's factor
static_assert(PADOC_E4M3_BF16_SHIFT_LOG2 == 112, "expansion factor");

struct DecodeParams {
    const int32_t *stream_page, *shared_len, *private_len, *slot_ptr;
    const int32_t *page_len;     // each page's shared-stream length (the plan's)
    // 1: the previous kernel in the stream is this step's append (padoc_mpd_launch_step), which
    // writes only each stream's newest row and the step's queries: warps of CTAs without
    // tensor-core work read their headers and block ids and start their first blocks (those
    // without a newest row) before they wait for it
    int32_t pre_wait;
    // with pre_wait (may be null): [num_warps][4] pool rows of the first four blocks of each warp's
    // first item (-2 - row: the block of its stream's newest row; -1 past its end), read beside the
    // item header instead of after it
    const int32_t *first_blocks;
    const padoc_item *items;
    int32_t first_item;          // warp items start here
    const int32_t *warp_ptr;     // warp w owns warp items [warp_ptr[w], warp_ptr[w+1])
    int32_t num_warps;
    const int32_t *page_table;
    const int32_t *stream_table;
    int32_t page_stride, stream_stride;
    int32_t num_blocks, num_kv_heads, num_q_heads, pool_rows;
    const __nv_bfloat16 *k_pool, *v_pool;
    const uint8_t *k_codes, *v_codes;     // E4M3 pool (k_pool / v_pool unused)
    const float *k_scales, *v_scales;
    const __nv_bfloat16 *q;
    __nv_bfloat16 *part_o;       // partial O, bf16 (workspace layout in plan_internal.h)
    float *part_lse;
    float scale_log2;
    int *err;
};

// One warp of the warp path: warp `warp` of its CTA (its ring starts at smem + warp x the ring
// size; smem is 1024-byte aligned) runs warp list wi < prm.num_warps, whole warp, no CTA barrier.
// kPreWait: the CTA has not waited for the previous kernel in the stream (prm.pre_wait): the warp
// waits itself once its first safe blocks are on the way.
template <bool kE4M3, bool kPreWait = false>
__device__ __forceinline__ void decode_warp_role(const DecodeParams &prm, uint8_t *smem, int warp, int lane, int wi)
{
    uint8_t *wbuf = smem + (size_t)warp * (kE4M3 ? kE8WarpBytes : kWarpRing);
    uint8_t *cbuf = wbuf + kWStages * kE8StageBytes;   // E4M3: the expanded bf16 block
    const padoc_item *items = prm.items + prm.first_item;
    const int i0 = prm.warp_ptr[wi], i1 = prm.warp_ptr[wi + 1];
    // Every global read the loop depends on is issued at least one item ahead: item headers two
    // items ahead, block ids (one per lane) and query fragments one item ahead, so a warp never
    // waits on a load between two paged blocks.
    auto load_item = [&](int u) { return items[u]; };   // 4-byte loads: the blob has no 16-byte alignment
    struct Walk {   // what the producer needs of an item
        const int32_t *table;
        int blk0, nblk, g;
    };
    auto walk_of = [&](const padoc_item &it) {
        Walk w;
        w.table = it.kind == PADOC_ITEM_SHARED ? prm.page_table + (size_t)it.index * prm.page_stride
                                               : prm.stream_table + (size_t)it.first_stream * prm.stream_stride;
        w.blk0 = it.tok_begin / kBlk;
        w.nblk = it.tok_end > it.tok_begin ? (it.tok_end - it.tok_begin + kBlk - 1) / kBlk : 0;
        w.g = it.kv_head;
        return w;
    };
    auto ids_of = [&](const Walk &w) { return lane < w.nblk ? w.table[w.blk0 + lane] : 0; };

    // The warp walks its items with one ring of kWStages paged blocks that runs on from one item
    // into the next. Producer: the next block to fetch is block pb of item pu (walk pc, ids ids_c);
    // item pu + 1 (walk pn, ids ids_n) and the header of item pu + 2 (hn2) are already on the way.
    // kPreWait with first_blocks: lane k < 4 holds the pool row of block k of the first item (>= 0),
    // -2 - that row for the block holding its stream's newest row, -1 past the item's end
    const bool have_fb = kPreWait && prm.first_blocks != nullptr;
    const int32_t fb = have_fb && lane < 4 ? prm.first_blocks[(size_t)wi * 4 + lane] : -1;
    int pu = i0, pb = 0;
    Walk pc{prm.page_table, 0, 0, 0}, pn{prm.page_table, 0, 0, 0};
    int32_t ids_c = 0, ids_n = 0;
    padoc_item hn2 = {};
    if (i0 < i1) { pc = walk_of(load_item(i0)); ids_c = ids_of(pc); }
    if (i0 + 1 < i1) { pn = walk_of(load_item(i0 + 1)); ids_n = ids_of(pn); }
    if (i0 + 2 < i1) hn2 = load_item(i0 + 2);
    const uint64_t kv_policy = l2_evict_first_policy();   // paged blocks are read once per call
    int ring = 0;   // blocks issued so far: block n goes to stage n % kWStages
    // chunk q = lane + 32k of a block's 512 16-byte chunks is panel q / 128 (K lo, K hi, V lo, V hi),
    // row (q / 8) % 16, 16-byte column q % 8 (swizzled)
    auto issue_next = [&]() {   // whole warp; always commits a group, possibly empty
        while (pu < i1 && pb >= pc.nblk) {
            ++pu;
            pb = 0;
            pc = pn;
            ids_c = ids_n;
            if (pu + 1 < i1) { pn = walk_of(hn2); ids_n = ids_of(pn); }
            if (pu + 2 < i1) hn2 = load_item(pu + 2);
        }
        if (pu < i1) {
            // block ids past the 32 a warp holds are read directly (the planner keeps items shorter)
            const int32_t id = pb < 32 ? __shfl_sync(0xffffffffu, ids_c, pb) : pc.table[pc.blk0 + pb];
            const bool okid = id >= 0 && id < prm.num_blocks;
            if (!okid && lane == 0) padoc_record_error(prm.err, PADOC_DEVERR_BLOCK_ID, id);
            const size_t rowbase = okid ? ((size_t)id * prm.num_kv_heads + pc.g) * kBlk : 0;
            if constexpr (kE4M3) {
                // chunk q = lane + 32k of the block's 256 16-byte chunks of codes: tensor q / 128,
                // row (q / 8) % 16, chunk q % 8 (swizzled by row); lanes 0 and 1 also copy the K and
                // V scales of the (block, KV head) (zeros for a bad id, whose codes are zeros too)
                const uint32_t base = smem_u32(wbuf + (ring % kWStages) * kE8StageBytes);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const int q = lane + 32 * k;
                    const int tn = q >> 7, r = (q >> 3) & 15, cc = q & 7;
                    const uint8_t *src = (tn == 0 ? prm.k_codes : prm.v_codes) + (rowbase + r) * kD + cc * 16;
                    cp_async_16_hint(base + tn * kE8Rows + r * 128 + ((cc ^ (r & 7)) << 4), src, okid ? 16u : 0u,
                                     kv_policy);
                }
                if (lane < 2) {
                    const size_t si = okid ? (size_t)id * prm.num_kv_heads + pc.g : 0;
                    cp_async_4(base + 2 * kE8Rows + lane * 4, (lane == 0 ? prm.k_scales : prm.v_scales) + si,
                               okid ? 4u : 0u);
                }
            } else {
                const uint32_t base = smem_u32(wbuf + (ring % kWStages) * kWStageBytes);
#pragma unroll
                for (int k = 0; k < 16; ++k) {
                    const int q = lane + 32 * k;
                    const int panel = q >> 7, r = (q >> 3) & 15, cc = q & 7;
                    const __nv_bfloat16 *src = (panel < 2 ? prm.k_pool : prm.v_pool) +
                                               (rowbase + r) * kD + (panel & 1) * 64 + cc * 8;
                    cp_async_16_hint(base + panel * kBoxBytes + r * 128 + ((cc ^ (r & 7)) << 4), src, okid ? 16u : 0u,
                                     kv_policy);
                }
            }
            ++pb;
            ++ring;
        }
        cp_async_commit();
    };
    int pre = 0;
    if constexpr (kPreWait) {
        // Before the wait: the first item's blocks ahead of the block holding its stream's newest
        // row (page_len - 1 of a shared item's page, private_len - 1 of a private item's stream),
        // which the append may be writing; everything read so far (plan, block tables) was copied
        // before the append started.
        if (have_fb) {
            // straight from the rows the host wrote, without waiting for the item header: the
            // leading blocks that exist, are in the pool and hold no newest row
            const bool ok = lane < 4 && fb >= 0 && fb <= prm.pool_rows - kBlk;
            const uint32_t okm = __ballot_sync(0xffffffffu, ok) & 0xfu;
            pre = min(__ffs(~okm) - 1, kWStages);
            for (int k = 0; k < pre; ++k) {
                const size_t rowbase = (size_t)__shfl_sync(0xffffffffu, fb, k);
                const uint32_t base = smem_u32(wbuf + k * kWStageBytes);
#pragma unroll
                for (int c = 0; c < 16; ++c) {
                    const int q = lane + 32 * c;
                    const int panel = q >> 7, r = (q >> 3) & 15, cc = q & 7;
                    const __nv_bfloat16 *src = (panel < 2 ? prm.k_pool : prm.v_pool) +
                                               (rowbase + r) * kD + (panel & 1) * 64 + cc * 8;
                    cp_async_16_hint(base + panel * kBoxBytes + r * 128 + ((cc ^ (r & 7)) << 4), src, 16u, kv_policy);
                }
                cp_async_commit();
            }
            pb = pre;
            ring = pre;
        } else if (i0 < i1) {
            const padoc_item it0 = load_item(i0);
            const int32_t len = it0.kind == PADOC_ITEM_SHARED ? prm.page_len[it0.index] : prm.private_len[it0.first_stream];
            pre = min(min(kWStages, pc.nblk), max(0, (len - 1) / kBlk - pc.blk0));
            for (int k = 0; k < pre; ++k) issue_next();
        }
        pdl_wait_prerequisite();
        pdl_launch_dependents();
    }
    for (int k = pre; k < kWStages; ++k) issue_next();

    // Consumer: header of the next item (ch_n) and of the one after (ch_n2), and the next item's
    // query fragments (B operand Q^T[128 dims x 8 heads]) and first partial row.
    padoc_item ch_n = {}, ch_n2 = {};
    uint32_t qn[8][2];
    size_t row_n = 0;
    auto load_q = [&](const padoc_item &it) {
        const __nv_bfloat16 *qrow =
            prm.q + ((size_t)it.first_stream * prm.num_q_heads + it.kv_head * kGroup + (lane >> 2)) * kD;
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
            qn[ks][0] = *reinterpret_cast<const uint32_t *>(qrow + ks * 16 + (lane & 3) * 2);
            qn[ks][1] = *reinterpret_cast<const uint32_t *>(qrow + ks * 16 + 8 + (lane & 3) * 2);
        }
        row_n = (size_t)(prm.slot_ptr[(size_t)it.first_stream * prm.num_kv_heads + it.kv_head] + it.slot) * kGroup;
    };
    if (i0 < i1) { ch_n = load_item(i0); load_q(ch_n); }
    if (i0 + 1 < i1) ch_n2 = load_item(i0 + 1);
    int gc = 0;   // blocks consumed so far
    for (int cu = i0; cu < i1; ++cu) {
        const padoc_item it = ch_n;
        uint32_t qb[8][2];
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) { qb[ks][0] = qn[ks][0]; qb[ks][1] = qn[ks][1]; }
        const size_t row0 = row_n;
        if (cu + 1 < i1) {
            ch_n = ch_n2;
            load_q(ch_n);
            if (cu + 2 < i1) ch_n2 = load_item(cu + 2);
        }
        const int cutoff = it.tok_end;   // the planner keeps warp items inside their stream's cutoff
        const int blk0 = it.tok_begin / kBlk;
        const int nblk = cutoff > it.tok_begin ? (cutoff - it.tok_begin + kBlk - 1) / kBlk : 0;
        float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};   // heads h0 = 2*(lane%4), h0+1
        float o[8][4];
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;

        for (int bi = 0; bi < nblk; ++bi, ++gc) {
            cp_async_wait<kWStages - 1>();   // block gc has landed (one group per block)
            __syncwarp();
            // per block: the multiplier of the raw scores (scale in log2 units) and, for an E4M3
            // pool, the factor folded into P (the V scale; both carry the expansion's 2^112)
            float kmul = prm.scale_log2, vfac = 1.f;
            uint32_t base;
            if constexpr (kE4M3) {
                const uint8_t *stg = wbuf + (gc % kWStages) * kE8StageBytes;
                const float ks = *reinterpret_cast<const float *>(stg + 2 * kE8Rows);
                const float vs = *reinterpret_cast<const float *>(stg + 2 * kE8Rows + 4);
                // a zero scale marks a block without a nonzero value (its codes are all zero):
                // any positive factor then gives the same scores and keeps masked ones at -inf
                kmul = prm.scale_log2 * (ks > 0.f ? ks : 1.f) * kTwo112;
                vfac = (vs > 0.f ? vs : 1.f) * kTwo112;
                // lane l expands row l % 16 of tensor l / 16 (K, V) into the bf16 panels
                const int tn = lane >> 4, r = lane & 15;
                uint4 raw[8];
#pragma unroll
                for (int c = 0; c < 8; ++c)
                    raw[c] = *reinterpret_cast<const uint4 *>(stg + tn * kE8Rows + r * 128 + ((c ^ (r & 7)) << 4));
                __syncwarp();   // every lane has its row: the stage may be refilled
                issue_next();
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    const uint32_t w[4] = {raw[c].x, raw[c].y, raw[c].z, raw[c].w};
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh) {   // dims 16c + 8hh .. + 7: bf16 chunk 2c + hh
                        const int k = 2 * c + hh, panel = 2 * tn + (k >> 3), kk = k & 7;
                        uint4 o;
                        o.x = e4m3x2_to_bf16x2_shifted((uint16_t)(w[2 * hh] & 0xFFFFu));
                        o.y = e4m3x2_to_bf16x2_shifted((uint16_t)(w[2 * hh] >> 16));
                        o.z = e4m3x2_to_bf16x2_shifted((uint16_t)(w[2 * hh + 1] & 0xFFFFu));
                        o.w = e4m3x2_to_bf16x2_shifted((uint16_t)(w[2 * hh + 1] >> 16));
                        *reinterpret_cast<uint4 *>(cbuf + panel * kBoxBytes + r * 128 + ((kk ^ (r & 7)) << 4)) = o;
                    }
                }
                __syncwarp();
                base = smem_u32(cbuf);
            } else {
                base = smem_u32(wbuf + (gc % kWStages) * kWStageBytes);
            }
            const int tokbase = (blk0 + bi) * kBlk;
            // S^T = K . Q^T, as two independent MMA chains (even / odd k-steps) added at the end
            float acc[4] = {0.f, 0.f, 0.f, 0.f}, acc2[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
                const uint32_t row = lane & 15;
                const uint32_t col = (ks & 3) * 16 + (lane >> 4) * 8;
                uint32_t a[4];
                ldmatrix_x4(a, base + (ks >> 2) * kBoxBytes + sw128_offset(row, col));
                mma_bf16_16816((ks & 1) ? acc2 : acc, a, qb[ks][0], qb[ks][1]);
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) acc[i] += acc2[i];
            const int t0 = tokbase + (lane >> 2), t1 = t0 + 8;
            float sc[4];
            sc[0] = t0 < cutoff ? acc[0] * kmul : -INFINITY;
            sc[1] = t0 < cutoff ? acc[1] * kmul : -INFINITY;
            sc[2] = t1 < cutoff ? acc[2] * kmul : -INFINITY;
            sc[3] = t1 < cutoff ? acc[3] * kmul : -INFINITY;
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
            const float r0 = mn0 == -INFINITY ? 0.f : mn0, r1 = mn1 == -INFINITY ? 0.f : mn1;
            const float p0 = fast_exp2(sc[0] - r0), p1 = fast_exp2(sc[1] - r1);
            const float p2 = fast_exp2(sc[2] - r0), p3 = fast_exp2(sc[3] - r1);
            m[0] = mn0; m[1] = mn1;
            l[0] = l[0] * al0 + p0 + p2;
            l[1] = l[1] * al1 + p1 + p3;
            // the V scale rides on P (E4M3); l keeps the plain probabilities
            const uint32_t b0 = movmatrix_trans(kE4M3 ? pack_bf16x2(p0 * vfac, p1 * vfac) : pack_bf16x2(p0, p1));
            const uint32_t b1 = movmatrix_trans(kE4M3 ? pack_bf16x2(p2 * vfac, p3 * vfac) : pack_bf16x2(p2, p3));
            if (__any_sync(0xffffffffu, al0 != 1.f || al1 != 1.f)) {   // a head's running max moved
#pragma unroll
                for (int mt = 0; mt < 8; ++mt) {
                    o[mt][0] *= al0; o[mt][1] *= al1; o[mt][2] *= al0; o[mt][3] *= al1;
                }
            }
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) {
                const int i = lane >> 3;
                const uint32_t row = (lane & 7) + (i >= 2 ? 8 : 0);
                const uint32_t col = (mt & 3) * 16 + (i & 1) * 8;
                uint32_t a[4];
                ldmatrix_x4_trans(a, base + (2 + (mt >> 2)) * kBoxBytes + sw128_offset(row, col));
                mma_bf16_16816(o[mt], a, b0, b1);
            }
            __syncwarp();   // every lane is done with the stage (bf16) or the expanded block (E4M3)
            if constexpr (!kE4M3) issue_next();   // (E4M3: the stage was refilled after its expansion)
        }
        // complete the row sums over the 8 token lanes of each head
#pragma unroll
        for (int sh = 4; sh < 32; sh <<= 1) {
            l[0] += __shfl_xor_sync(0xffffffffu, l[0], sh);
            l[1] += __shfl_xor_sync(0xffffffffu, l[1], sh);
        }
        // the partial in bf16, in the slot layout [16 chunks of 8 dims][8 heads][8]: lane l holds dim
        // l / 4 of heads h0, h0 + 1 (h0 = 2 (l % 4)); with its partner l ^ 4 (the next or previous dim)
        // a lane of an even dim writes the dim pair of head h0, one of an odd dim that of head
        // h0 + 1, so that the warp writes each chunk's [8 heads][8 dims] as one 128-byte run
        {
            const int h0 = (lane & 3) * 2, dm = lane >> 2;
            const bool ev = (dm & 1) == 0;
            const float i0f = l[0] > 0.f ? 1.f / l[0] : 0.f, i1f = l[1] > 0.f ? 1.f / l[1] : 0.f;
            // element offset of this lane's pair inside a chunk
            const int off = ev ? h0 * 8 + dm : (h0 + 1) * 8 + dm - 1;
            uint32_t *p = reinterpret_cast<uint32_t *>(prm.part_o + row0 * kD);   // row0 = slot * 8
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) {
#pragma unroll
                for (int c = 0; c < 2; ++c) {   // chunk 2 mt + c: registers 2c (head h0), 2c + 1 (h0 + 1)
                    const float a = o[mt][2 * c] * i0f, b = o[mt][2 * c + 1] * i1f;
                    const float pa = __shfl_xor_sync(0xffffffffu, a, 4), pb = __shfl_xor_sync(0xffffffffu, b, 4);
                    p[((2 * mt + c) * 64 + off) >> 1] = ev ? pack_bf16x2(a, pa) : pack_bf16x2(pb, b);
                }
            }
        }
        if (lane < 4) {
            const int h0 = lane * 2;
            prm.part_lse[row0 + h0] = l[0] > 0.f ? (m[0] + log2f(l[0])) * PADOC_LN2 : -INFINITY;
            prm.part_lse[row0 + h0 + 1] = l[1] > 0.f ? (m[1] + log2f(l[1])) * PADOC_LN2 : -INFINITY;
        }
    }
    cp_async_wait<0>();
}

}  // namespace padoc_warp
