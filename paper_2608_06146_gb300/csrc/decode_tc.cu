// decode_tc.cu -- C2 on the 5th-generation tensor cores: the shared-stream part of one decode step.
//
// For a page whose branches x query heads (of one KV head) fill dense M = 128 tiles, the page's
// shared stream (prefix + layout, stored once in the paged KV cache) is read once per K/V tile of
// 128 tokens and multiplied against the queries of up to 32 of its streams: two M-tiles of 16
// streams x 8 query heads. Row (stream b, head h) sees the columns before its own cutoff P + f_k
// (Algorithm 1's mask row restricted to the shared stream).
//
// The kernel is persistent and stream-K balanced: the planner lays every (KV head, page, stream
// group) tile sequence end to end and gives each CTA one contiguous range of equal work, which
// becomes a list of pieces (a piece = the tiles of one sequence inside the range). A CTA walks its
// pieces back to back; its K/V ring, barrier phases and TMEM carry over from one piece to the next,
// so the next piece's tiles are in flight while the current one finishes. Each piece writes one
// partial (normalized O, natural-log LSE) per (stream, head) into its split-K slot; the merge
// kernel joins the partials of a (stream, KV head).
//
// CTA layout: warps 0-7 run the softmax and epilogue of one M-tile at a time (M-tile 0, then 1,
// tile by tile): warp w reads TMEM lanes 32 (w % 4) ... (one row per thread) and column half w / 4,
// and the two threads of a row swap their partial row max (and, at the end, row sum) through
// shared memory. While they work on one M-tile, the tensor cores run the other M-tile's PV and
// next QK^T. Warps 8 and 10 are the TMA producers of the K ring (3 tiles: a K tile is free once
// its QK^T completes, so K runs two tiles ahead) and the V ring (2 tiles: V is held until the
// tile's PV completes): lanes 0-7 each fetch one 16-token paged block per tile, two 64-column boxes,
// with the block ids looked up one tile ahead; blocks past the piece or with an out-of-range id are
// fetched from an out-of-range coordinate, which fills zeros. Warp 8 also fetches each piece's
// queries (one 4-D box per panel) once the previous piece's last QK^T has completed. Warp 9
// allocates TMEM; warps 9 and 11 issue the MMAs of M-tile 0 and M-tile 1, each as a converged warp.
// TMEM: S_i / P_i at columns 128i, O_i at 256 + 128i. The next piece's first PV overwrites O_i; it
// waits for P_i of that piece, which the softmax warps publish only after reading O_i out.
//
// A piece may span two items (chunked prefill: a group's shared tiles, then its private ones; the
// first item flagged PADOC_ITEM_CONT): the second item keeps the queries, the softmax state and O
// (its first PV accumulates), and only it writes the partial.
//
// FP8 (E4M3) pool (kE4M3): each paged block's codes (16 rows x 128 bytes) land by TMA in the upper
// half of the tile's ring slot, and the producer warp that loaded them expands them in place into
// the bf16 panels the MMAs read (each lane owns whole rows, reads a row's codes before writing it;
// codes times 2^-112 are exact bf16 values), then marks the slot full. A producer expands tile n - 2
// (K) or n - 1 (V) before it issues tile n, so loads stay in flight while it converts. The K
// producer also copies each block's K and V scales into a ring of 8 entries, one per tile; the
// softmax applies the K scale to the block's scores and folds the V scale into the block's
// probabilities before they are rounded to bf16, and removes it again from their row sum.
#include <math.h>

#include "common.cuh"
#include "decode_warp.cuh"
#include "tc.cuh"

namespace {

constexpr int kD = 128;
constexpr int kGroup = 8;        // query heads per KV head
constexpr int kBlk = 16;         // tokens per paged block
constexpr int kKT = 128;         // tokens per K/V tile
constexpr int kPanel = 128 * 128;
constexpr int kTile = 2 * kPanel;
constexpr int kKStages = 3;       // K tiles in the ring: K is released early (after QK^T)
constexpr int kVStages = 2;       // V tiles in the ring: V is held until the tile's PV completes
constexpr uint32_t kTmemCols = 512;
constexpr int kThreads = 384;

enum {
    B_Q = 0,         // the piece's queries have landed
    B_QFREE = 1,     // the piece's last QK^T has completed: the query buffer may be refilled
    B_KFULL = 2,     // [K stage]
    B_KEMPTY = 5,    // [K stage]: the last QK^T of the tile has completed
    B_VFULL = 8,     // [V stage]
    B_VEMPTY = 10,   // [V stage]: the last PV of the tile has completed
    B_SFULL = 12,    // [m-tile]
    B_PFULL = 14,    // [m-tile], one arrival per softmax warp
    B_PVDONE = 16,   // [m-tile]: the piece's last PV has completed (O_i is final)
    B_FINAL = 18,
    B_KSTG = 19,     // [K stage] E4M3: the tile's codes have landed
    B_VSTG = 22,     // [V stage] E4M3
    B_SCL = 24,      // [scale entry] E4M3: the tile's scales have landed (one arrival per loading lane)
    B_COUNT = 32
};
constexpr int kSclEntries = 8;   // scale ring: entry n % 8 for tile n

constexpr int kSoftmaxWarps = 8;
constexpr int kXchBytes = 2 * 2 * 128 * 4;   // row max / sum swap: [buffer][column half][row] floats
// Q (two M-tiles), the K and V rings, then barriers (256 bytes), the TMEM address and abort flag,
// the scale ring (E4M3: [8 entries][8 K scales, 8 V scales]) and the swap buffer: 232,448 bytes,
// the most a CTA may have, so there is no room to align the start by hand; the kernel checks that
// the driver placed it on a 1024-byte boundary (the base of a CTA's dynamic shared memory is) and
// refuses to run otherwise.
constexpr size_t kTilesBytes = (size_t)kTile * (2 + kKStages + kVStages);
constexpr int kMiscScl = 320, kMiscXch = 1024;
constexpr size_t kSmemBytes = kTilesBytes + kMiscXch + kXchBytes;
static_assert(kSmemBytes <= 232448, "shared memory per CTA");
static_assert(B_COUNT * 8 <= 256 && kMiscScl + kSclEntries * 16 * 4 <= kMiscXch, "misc layout");
constexpr float kTwo112 = 5.192296858534828e33f;   // 2^112: the bf16 expansion's factor
static_assert(PADOC_E4M3_BF16_SHIFT_LOG2 == 112, "expansion factor");

struct TcDecodeParams {
    const int32_t *shared_len, *private_len, *slot_ptr, *cta_ptr;
    const padoc_item *items;
    int32_t num_tc_items, num_pages, num_streams;
    const int32_t *page_table, *stream_table;
    int32_t page_stride, stream_stride;
    int32_t num_blocks, num_kv_heads;
    int32_t pool_rows;           // num_blocks * num_kv_heads * 16: first out-of-range row
    const float *k_scales, *v_scales;   // E4M3 pool: [num_blocks][num_kv_heads]
    __nv_bfloat16 *part_o;       // partial O, bf16 (workspace layout in plan_internal.h)
    float *part_lse;
    __nv_bfloat16 *out;          // [S][Hq][128]: written directly by PADOC_ITEM_SOLE items
    float *lse;                  // [S][Hq]
    int32_t num_q_heads;
    float scale_log2;
    int *err;
    // the fused grid (plan_internal.h): CTAs [0, tc_ctas) run pieces, then warp CTA early_ctas + c;
    // CTAs from tc_ctas on run warp CTA c - tc_ctas; warp CTAs at or past warp_ctas do not exist
    int32_t tc_ctas, early_ctas, warp_ctas;
};

__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, int *err, int site, volatile int *abort_flag)
{
    if (*abort_flag) return false;
    if (mbar_wait_bounded(bar, parity, err, site)) return true;
    *abort_flag = 1;
    return false;
}

__device__ __forceinline__ int piece_tiles(const padoc_item &it)
{
    return it.tok_end > it.tok_begin ? (it.tok_end - it.tok_begin + kKT - 1) / kKT : 0;
}

__device__ __forceinline__ int piece_mtiles(const padoc_item &it) { return it.num_streams > 16 ? 2 : 1; }

// The block-table row an item walks: a page's shared stream (PADOC_ITEM_SHARED_TC, index = page) or
// the private rows of a chunk of one stream's consecutive query tokens (PADOC_ITEM_PRIVATE_TC, index
// = the chunk's first stream, whose row every token of the chunk shares). Returns null when the
// row is out of range.
__device__ __forceinline__ const int32_t *item_row(const TcDecodeParams &prm, const padoc_item &it, int32_t &stride)
{
    const bool priv = PADOC_ITEM_KIND(it.kind) == PADOC_ITEM_PRIVATE_TC;
    stride = priv ? prm.stream_stride : prm.page_stride;
    const int32_t rows = priv ? prm.num_streams : prm.num_pages;
    if (it.index < 0 || it.index >= rows) return nullptr;
    return (priv ? prm.stream_table : prm.page_table) + (size_t)it.index * stride;
}

// E4M3: expands one landed tile of codes in place into the slot's two bf16 panels. Lane l owns
// rows l, l + 32, l + 64, l + 96; it reads a row's eight 16-byte chunks of codes (swizzled by row,
// in the upper half of the slot, where the row's panel-1 bytes go) before it writes the row.
__device__ __forceinline__ void expand_tile(uint8_t *slot, int lane)
{
    const uint8_t *codes = slot + kPanel;
#pragma unroll 1
    for (int k = 0; k < 4; ++k) {
        const int r = lane + 32 * k;
        uint4 raw[8];
#pragma unroll
        for (int c = 0; c < 8; ++c) raw[c] = *reinterpret_cast<const uint4 *>(codes + r * 128 + ((c ^ (r & 7)) << 4));
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            const uint32_t w[4] = {raw[c].x, raw[c].y, raw[c].z, raw[c].w};
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {   // dims 16c + 8hh .. + 7: chunk 2c + hh of the row
                const int kk = 2 * c + hh;
                uint4 o;
                o.x = e4m3x2_to_bf16x2_shifted((uint16_t)(w[2 * hh] & 0xFFFFu));
                o.y = e4m3x2_to_bf16x2_shifted((uint16_t)(w[2 * hh] >> 16));
                o.z = e4m3x2_to_bf16x2_shifted((uint16_t)(w[2 * hh + 1] & 0xFFFFu));
                o.w = e4m3x2_to_bf16x2_shifted((uint16_t)(w[2 * hh + 1] >> 16));
                *reinterpret_cast<uint4 *>(slot + (kk >> 3) * kPanel + r * 128 + (((kk & 7) ^ (r & 7)) << 4)) = o;
            }
        }
    }
    fence_proxy_async_smem();   // the MMAs read the panels through the async proxy
}

// Pulls into L2 the first paged blocks (up to 4) of the first item of each of warp CTA wc's warp
// lists, which this CTA runs once its pieces end, so that they land from L2 rather than from a
// memory system under full load. Lane l takes block l % 4 of warp l / 4's first item; it reads the
// same plan words and block-table entries that warp reads, and skips out-of-range block ids.
template <bool kE4M3>
__device__ __forceinline__ void prefetch_warp_lists(const padoc_warp::DecodeParams &w, const CUtensorMap &kmap,
                                                    const CUtensorMap &vmap, int wc, int lane)
{
    const int wi = wc * padoc_warp::kWarps + (lane >> 2), b = lane & 3;
    if (wi >= w.num_warps) return;
    const int i0 = w.warp_ptr[wi], i1 = w.warp_ptr[wi + 1];
    if (i0 >= i1) return;
    const padoc_item it = w.items[w.first_item + i0];
    const int tok = it.tok_begin + b * kBlk;
    if (tok >= it.tok_end) return;
    const int32_t *table = it.kind == PADOC_ITEM_SHARED ? w.page_table + (size_t)it.index * w.page_stride
                                                        : w.stream_table + (size_t)it.first_stream * w.stream_stride;
    const int32_t id = table[tok / kBlk];
    if (id < 0 || id >= w.num_blocks) return;
    const int32_t row = (id * w.num_kv_heads + it.kv_head) * kBlk;
    tma_prefetch_l2_2d(&kmap, 0, row);
    tma_prefetch_l2_2d(&vmap, 0, row);
    if (!kE4M3) {   // (an E4M3 box holds the whole row)
        tma_prefetch_l2_2d(&kmap, 64, row);
        tma_prefetch_l2_2d(&vmap, 64, row);
    }
}

// The pieces of tensor-core CTA blockIdx.x (every thread of the CTA; smem 1024-byte aligned).
// kFused: the CTA runs warp lists next (their first blocks are pulled into L2 meanwhile). kSole:
// the plan has PADOC_ITEM_SOLE items (otherwise their output path is compiled out).
template <bool kE4M3, bool kFused, bool kSole>
__device__ __forceinline__ void decode_tc_role(const CUtensorMap &kmap, const CUtensorMap &vmap, const CUtensorMap &qmap,
                                               const TcDecodeParams &prm, const padoc_warp::DecodeParams &wprm,
                                               uint8_t *smem)
{
    uint8_t *sq = smem;
    uint8_t *sk = sq + 2 * kTile;
    uint8_t *sv = sk + kKStages * kTile;
    uint8_t *misc = smem + kTilesBytes;
    uint64_t *bars = (uint64_t *)misc;
    uint32_t *tmem_slot = (uint32_t *)(misc + 256);
    volatile int *abort_flag = (volatile int *)(misc + 260);
    float *scl = (float *)(misc + kMiscScl);   // E4M3: [entry][K scales of 8 blocks, V scales of 8 blocks]
    float *xch = (float *)(misc + kMiscXch);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar = [&](int i) { return smem_u32(&bars[i]); };
    if (warp == 8 || warp == 10) {
        // Before this grid waits for the previous kernel, the producers pull the CTA's first queries
        // and first two K/V tiles into L2. L2 is where every write lands, so a prefetch can only
        // warm it, never serve stale data later; every index is range-checked first, and a tensor
        // prefetch past the pool fetches nothing.
        const int a0 = prm.cta_ptr[blockIdx.x], a1 = prm.cta_ptr[blockIdx.x + 1];
        if (a0 >= 0 && a0 < a1 && a0 < prm.num_tc_items) {
            const padoc_item it = prm.items[a0];
            const CUtensorMap *map = warp == 8 ? &kmap : &vmap;
            const int j = lane >> 3, b = lane & 7;   // lanes 0-15: tiles 0-1, blocks 0-7
            const int tok0 = it.tok_begin + j * kKT + b * kBlk;
            int32_t stride = 0;
            const int32_t *trow = item_row(prm, it, stride);
            if (lane < 16 && trow && tok0 >= 0 && tok0 < it.tok_end && tok0 / kBlk < stride) {
                const int32_t id = trow[tok0 / kBlk];
                if (id >= 0 && id < prm.num_blocks) {
                    const int32_t row = (id * prm.num_kv_heads + it.kv_head) * kBlk;
                    tma_prefetch_l2_2d(map, 0, row);
                    if (!kE4M3) tma_prefetch_l2_2d(map, 64, row);   // (an E4M3 box holds the whole row)
                }
            }
            if (warp == 8 && lane == 16)
                for (int i = 0; i < piece_mtiles(it); ++i) {
                    tma_prefetch_l2_4d(&qmap, 0, 0, it.kv_head, it.first_stream + 16 * i);
                    tma_prefetch_l2_4d(&qmap, 64, 0, it.kv_head, it.first_stream + 16 * i);
                }
        }
    }
    if (tid == 0) {
        for (int i = 0; i < B_COUNT; ++i)
            mbar_init(smem_u32(&bars[i]), (i == B_PFULL || i == B_PFULL + 1) ? kSoftmaxWarps
                                          : (i == B_QFREE || (i >= B_KEMPTY && i < B_KEMPTY + kKStages) ||
                                             (i >= B_VEMPTY && i < B_VEMPTY + kVStages) || i == B_FINAL)
                                                ? 2     // one commit from each MMA warp
                                          : (i >= B_SCL) ? kKT / kBlk   // one per lane that loads a block
                                                : 1);
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
    // Nothing above touches global memory, so under a programmatic launch it overlaps the end of
    // the previous kernel in the stream. From here on the grid reads its inputs and writes partials
    // (which the previous step's merge may still be reading), so it first waits for that kernel, and
    // only then lets the warp kernel (which writes partials too) launch.
    pdl_wait_prerequisite();
    pdl_launch_dependents();
    const int u0 = prm.cta_ptr[blockIdx.x], u1 = prm.cta_ptr[blockIdx.x + 1];

    if (warp == 8 || warp == 10) {
        // ---------------------------------------------------------------- TMA producers (whole warps)
        // warp 8 fills the K ring (and loads each piece's queries), warp 10 the V ring, each as far
        // ahead as its ring allows. Lane l < 8 owns paged block l of every tile; its block id is read
        // one tile ahead.
        const bool is_k = warp == 8;
        const int nst = is_k ? kKStages : kVStages;
        const CUtensorMap *map = is_k ? &kmap : &vmap;
        uint8_t *ring = is_k ? sk : sv;
        const int b_full = is_k ? B_KFULL : B_VFULL, b_empty = is_k ? B_KEMPTY : B_VEMPTY;
        // K/V tiles read by one group only are evict-first; see PADOC_ITEM_REREAD
        const uint64_t once_policy = l2_evict_first_policy(), shared_policy = l2_evict_normal_policy();
        int32_t id_next = 0;
        bool in_next = false;
        auto fetch_id = [&](int uu, int jj) {
            const padoc_item &p = prm.items[uu];
            const int tok0 = p.tok_begin + jj * kKT + lane * kBlk;
            int32_t stride = 0;
            const int32_t *trow = item_row(prm, p, stride);
            in_next = lane < kKT / kBlk && tok0 < p.tok_end;
            // a table row or block index the plan never produces reads as block -1, which the range
            // check below reports and skips
            id_next = !in_next ? 0 : (trow != nullptr && tok0 / kBlk < stride) ? trow[tok0 / kBlk] : -1;
        };
        // a piece's queries: one 4-D box per 64-column panel gathers 16 streams x the 8 heads of the
        // KV head; the next piece's boxes are pulled into L2 meanwhile, so that its reload (which
        // must wait for this piece's last QK^T) is short
        auto load_q = [&](const padoc_item &p, int uu) {
            const int mt = piece_mtiles(p);
            mbar_arrive_expect_tx(bar(B_Q), mt * kTile);
            for (int i = 0; i < mt; ++i) {
                tma_load_4d(smem_u32(sq + i * kTile), &qmap, 0, 0, p.kv_head, p.first_stream + 16 * i, bar(B_Q));
                tma_load_4d(smem_u32(sq + i * kTile) + kPanel, &qmap, 64, 0, p.kv_head, p.first_stream + 16 * i, bar(B_Q));
            }
            if (uu + 1 < u1) {
                const padoc_item &n = prm.items[uu + 1];
                for (int i = 0; i < piece_mtiles(n); ++i) {
                    tma_prefetch_l2_4d(&qmap, 0, 0, n.kv_head, n.first_stream + 16 * i);
                    tma_prefetch_l2_4d(&qmap, 64, 0, n.kv_head, n.first_stream + 16 * i);
                }
            }
        };
        if (u0 < u1) fetch_id(u0, 0);
        int n = 0, nq = 0;   // tiles and query sets issued
        // E4M3: tiles expanded so far; a tile is expanded `lag` tiles after it is issued (K runs
        // further ahead: its ring has three slots)
        int nc = 0;
        const int lag = is_k ? 2 : 1;
        const int b_stg = is_k ? B_KSTG : B_VSTG;
        auto expand_next = [&]() {   // whole warp; nc counts only tiles whose codes have landed
            const int t = nc;
            const int st = t % nst;
            bool r = wait_or_abort(bar(b_stg + st), (t / nst) & 1, prm.err, is_k ? 56 : 57, abort_flag);
            r = __all_sync(0xffffffffu, r);
            if (!r) return false;
            ++nc;
            expand_tile(ring + st * kTile, lane);
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(b_full + st));
            return true;
        };
        // the first piece's queries go out before anything else (they wait for nothing)
        const bool q_first = is_k && u0 < u1 && piece_tiles(prm.items[u0]) > 0;
        if (q_first) {
            if (lane == 0) load_q(prm.items[u0], u0);
            nq = 1;
        }
        bool ok = true;
        for (int u = u0; ok && u < u1; ++u) {
            const padoc_item it = prm.items[u];
            const int ne = piece_tiles(it);
            // an item that continues the previous one keeps its queries
            const bool cont_in = u > u0 && (prm.items[u - 1].kind & PADOC_ITEM_CONT);
            if (ne == 0) {
                if (u + 1 < u1) fetch_id(u + 1, 0);
                continue;
            }
            for (int j = 0; j < ne; ++j) {
                const int32_t id = id_next;
                const bool in = in_next;
                if (j + 1 < ne) fetch_id(u, j + 1);
                else if (u + 1 < u1) fetch_id(u + 1, 0);
                int32_t row = prm.pool_rows;
                if (in) {
                    if (id >= 0 && id < prm.num_blocks) row = (id * prm.num_kv_heads + it.kv_head) * kBlk;
                    else if (is_k) padoc_record_error(prm.err, PADOC_DEVERR_BLOCK_ID, id);
                }
                const int s = n % nst, use = n / nst;
                if (kE4M3)
                    while (ok && nc <= n - lag) ok = expand_next();
                if (!ok) break;
                if (use > 0) ok = wait_or_abort(bar(b_empty + s), (use - 1) & 1, prm.err, is_k ? 50 : 53, abort_flag);
                if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
                const uint64_t kv_policy = (it.kind & PADOC_ITEM_REREAD) ? shared_policy : once_policy;
                if constexpr (kE4M3) {
                    // the block's codes (16 rows x 128 bytes) into the slot's upper half; the K warp also
                    // copies the block's two scales into the tile's scale entry (zeros past the piece
                    // or for a bad id, whose codes are zeros too)
                    if (lane == 0) mbar_arrive_expect_tx(bar(b_stg + s), kTile / 2);
                    __syncwarp();
                    if (lane < kKT / kBlk) {
                        const uint32_t dst = smem_u32(ring + s * kTile) + kPanel + (uint32_t)lane * (kBlk * 128);
                        tma_load_2d_hint(dst, map, 0, row, bar(b_stg + s), kv_policy);
                        if (is_k) {
                            const bool okid = row != prm.pool_rows;
                            const size_t si = okid ? (size_t)id * prm.num_kv_heads + it.kv_head : 0;
                            float *e = scl + (n % kSclEntries) * 16;
                            cp_async_4(smem_u32(e + lane), prm.k_scales + si, okid ? 4u : 0u);
                            cp_async_4(smem_u32(e + 8 + lane), prm.v_scales + si, okid ? 4u : 0u);
                            cp_async_mbar_arrive(bar(B_SCL + n % kSclEntries));
                        }
                    }
                } else {
                    if (lane == 0) mbar_arrive_expect_tx(bar(b_full + s), kTile);
                    __syncwarp();
                    if (lane < kKT / kBlk) {
                        const uint32_t dst = smem_u32(ring + s * kTile) + (uint32_t)lane * (kBlk * 128);
                        tma_load_2d_hint(dst, map, 0, row, bar(b_full + s), kv_policy);
                        tma_load_2d_hint(dst + kPanel, map, 64, row, bar(b_full + s), kv_policy);
                    }
                }
                ++n;
                if (is_k && j == 0 && !(q_first && u == u0) && !cont_in) {
                    // E4M3: the previous piece's tiles must be expanded before its last QK^T can run
                    if (kE4M3)
                        while (ok && nc < n - 1) ok = expand_next();
                    if (!ok) break;
                    // this piece's queries, once the previous piece's last QK^T has read the buffer
                    if (nq > 0) ok = wait_or_abort(bar(B_QFREE), (nq - 1) & 1, prm.err, 55, abort_flag);
                    if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
                    if (lane == 0) load_q(it, u);
                    ++nq;
                }
            }
        }
        // the K producer is done first (its ring runs two tiles ahead): it warms L2 for the warp lists
        // this CTA runs next (E4M3: after the last expansions below)
        const int wc = prm.early_ctas + (int)blockIdx.x;
        if (kFused && !kE4M3 && is_k && wc < prm.warp_ctas) prefetch_warp_lists<kE4M3>(wprm, kmap, vmap, wc, lane);
        if constexpr (kE4M3) {
            // the last tiles' expansion; after a failed wait only their copies are waited for
            while (ok && nc < n) ok = expand_next();
            if (kFused && is_k && wc < prm.warp_ctas) prefetch_warp_lists<kE4M3>(wprm, kmap, vmap, wc, lane);
            if (lane == 0)
                for (int J = nc; J < n; ++J)
                    mbar_wait_bounded(bar(b_stg + J % nst), (J / nst) & 1, prm.err, is_k ? 51 : 52);
            if (is_k) cp_async_wait<0>();
            if (lane == 0 && nq > 0) mbar_wait_bounded(bar(B_Q), (nq - 1) & 1, prm.err, 54);
        } else if (lane == 0) {
            // copies still in flight must land before the CTA's shared memory is released
            if (nq > 0) mbar_wait_bounded(bar(B_Q), (nq - 1) & 1, prm.err, 54);
            for (int J = (n > nst ? n - nst : 0); J < n; ++J)
                mbar_wait_bounded(bar(b_full + J % nst), (J / nst) & 1, prm.err, is_k ? 51 : 52);
        }
    } else if (warp == 9 || warp == 11) {
        // ---------------------------------------------------------------- MMA issuers (whole warps)
        // warp 9 issues M-tile 0's MMAs and warp 11 M-tile 1's, so that the waits, fences and
        // commits of one chain (each costs the issuing warp ~200 cycles) overlap the other chain's
        // MMAs on the tensor pipe. Both commit to the K/V-release, query-release and final
        // barriers (two arrivals each); on a one-M-tile piece warp 11 only commits.
        const int mi = warp == 9 ? 0 : 1;
        constexpr uint32_t idS = umma_idesc_bf16(128, kKT, false);
        constexpr uint32_t idPV = umma_idesc_bf16(128, kD, true);
        const uint64_t dq = umma_desc_sw128(smem_u32(sq + mi * kTile), 16, 1024);
        // stage descriptors differ only in the start-address field (address >> 4)
        const uint64_t dk0 = umma_desc_sw128(smem_u32(sk), 16, 1024);
        const uint64_t dv0 = umma_desc_sw128(smem_u32(sv), kPanel, 1024);
        const uint32_t tS = tmem + 128 * mi, tO = tmem + 256 + 128 * mi;
        auto wait_w = [&](int b, uint32_t parity, int site) {
            const bool r = wait_or_abort(bar(b), parity, prm.err, site, abort_flag);
            return __all_sync(0xffffffffu, r);
        };
        auto issue_s = [&](int stage) {
            const uint64_t db = dk0 + (uint64_t)(stage * (kTile >> 4));
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
                const uint32_t off = ((ks >> 2) * kPanel + (ks & 3) * 32) >> 4;
                umma_bf16_ss_warp(tS, dq + off, db + off, idS, ks > 0);
            }
            umma_commit_warp(bar(B_SFULL + mi));
        };
        int J = 0, nq = 0, ci = 0;   // tiles done, query sets used, tiles of this M-tile
        bool ok = true;
        for (int u = u0; ok && u < u1; ++u) {
            const padoc_item it = prm.items[u];
            const int ne = piece_tiles(it);
            const bool act = mi < piece_mtiles(it);   // this warp's M-tile is part of the piece
            // a piece over two items: the second keeps the queries and accumulates into O; only the
            // last item of a piece releases the queries and reports O complete
            const bool cont_in = u > u0 && (prm.items[u - 1].kind & PADOC_ITEM_CONT);
            const bool cont_out = (it.kind & PADOC_ITEM_CONT) != 0;
            if (ne == 0) continue;
            if ((!cont_in && !wait_w(B_Q, nq & 1, 60)) || !wait_w(B_KFULL + J % kKStages, (J / kKStages) & 1, 61)) {
                ok = false;
                break;
            }
            if (!cont_in) ++nq;
            tc_fence_after();
            if (act) issue_s(J % kKStages);
            umma_commit_warp(bar(B_KEMPTY + J % kKStages));
            if (ne == 1 && !cont_out) umma_commit_warp(bar(B_QFREE));
            for (int j = 0; ok && j < ne; ++j) {
                const int Jj = J + j, s = Jj % kVStages, kn = (Jj + 1) % kKStages;
                const bool more = j + 1 < ne;
                // The tile's V and the next K landed long before the softmax publishes P, so their
                // waits come first; between P and the next QK^T there is then one wait, one fence
                // and the MMAs, and every release is committed after them. (An idle warp still
                // waits for each tile it releases, so it never arrives twice on one phase.)
                if (!wait_w(B_VFULL + s, (Jj / kVStages) & 1, 63) ||
                    (more && !wait_w(B_KFULL + kn, ((Jj + 1) / kKStages) & 1, 64))) { ok = false; break; }
                if (act) {
                    if (!wait_w(B_PFULL + mi, ci & 1, 62)) { ok = false; break; }
                    tc_fence_after();
                    const uint64_t db = dv0 + (uint64_t)(s * (kTile >> 4));
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk)
                        umma_bf16_ts_warp(tO, tS + kk * 8, db + kk * (2048 >> 4), idPV, (cont_in || j > 0 || kk > 0));
                    ++ci;
                    // S_i of the next tile overwrites P_i only after this PV has read it (one
                    // thread's MMAs run in issue order)
                    if (more) issue_s(kn);
                    else if (!cont_out) umma_commit_warp(bar(B_PVDONE + mi));   // O_i of the piece is complete
                }
                umma_commit_warp(bar(B_VEMPTY + s));
                if (more) {
                    umma_commit_warp(bar(B_KEMPTY + kn));
                    if (j + 2 == ne && !cont_out) umma_commit_warp(bar(B_QFREE));
                }
            }
            J += ne;
        }
        // every MMA issued above must complete before TMEM is released
        umma_commit_warp(bar(B_FINAL));
        mbar_wait_bounded(bar(B_FINAL), 0, prm.err, 65);
    } else {
        // ---------------------------------------------------------------- softmax and epilogue
        const int quad = warp & 3, hc = warp >> 2;   // TMEM lane quarter, column half
        const int row = quad * 32 + lane;            // row of the M-tile = TMEM lane
        const int hl = row % kGroup;
        const uint32_t lanes = (uint32_t)(quad * 32) << 16;
        const float c = prm.scale_log2;
        const float cm = kE4M3 ? 1.f : c;   // E4M3: the row maxima are already scaled by the multipliers
        auto wait_all = [&](int bb, uint32_t parity, int site) {
            const bool r = wait_or_abort(bar(bb), parity, prm.err, site, abort_flag);
            return __all_sync(0xffffffffu, r);
        };
        // Warps w and w + 4 (the same TMEM lanes, the two column halves) meet at a named barrier of
        // their own (1 + w % 4) for every swap, so neither may leave the loops early: after a failed
        // wait (ok = false) a warp skips the work but still takes every swap.
        int nx = 0;   // row-value swaps so far (double-buffered)
        auto swap_row = [&](float v) {   // returns the value the other column half passed for this row
            float *buf = xch + (nx & 1) * 256;
            buf[hc * 128 + row] = v;
            named_bar_sync(1 + quad, 64);
            const float o = buf[(hc ^ 1) * 128 + row];
            ++nx;
            return o;
        };
        int cnt0 = 0, cnt1 = 0;   // tiles of M-tile 0 / 1 so far
        int pd0 = 0, pd1 = 0;     // pieces of M-tile 0 / 1 with tiles so far
        bool ok = true;
        // The next piece's fields are read while the current piece runs (its item at the piece's
        // start, the rows' cutoffs after its first tile), so no global load latency sits between
        // two pieces. Rows (stream b = 16 mi + row / 8, head row % 8) of M-tile mi see the shared
        // columns before their cutoff.
        const int b0 = row / kGroup, b1 = 16 + row / kGroup;
        int n_tb = 0, n_te = 0, n_nstr = 0, n_first = 0, n_kvh = 0, n_slot = 0, n_cut0 = 0, n_cut1 = 0;
        bool n_priv = false, n_cont = false, n_sole = false;
        auto fetch_item = [&](int uu) {
            const padoc_item *p = prm.items + uu;
            n_tb = p->tok_begin;
            n_te = p->tok_end;
            n_nstr = p->num_streams;
            n_first = p->first_stream;
            n_kvh = p->kv_head;
            n_slot = p->slot;
            n_priv = PADOC_ITEM_KIND(p->kind) == PADOC_ITEM_PRIVATE_TC;
            n_cont = (p->kind & PADOC_ITEM_CONT) != 0;
            n_sole = (p->kind & PADOC_ITEM_SOLE) != 0;
        };
        // a row's cutoff: its stream's shared length, or for a chunk's private rows its private length
        auto fetch_cut = [&]() {
            const int32_t *cut = n_priv ? prm.private_len : prm.shared_len;
            n_cut0 = b0 < n_nstr ? min(cut[n_first + b0], n_te) : n_tb;
            n_cut1 = b1 < n_nstr ? min(cut[n_first + b1], n_te) : n_tb;
        };
        if (u0 < u1) {
            fetch_item(u0);
            fetch_cut();
        }
        float m0 = -INFINITY, l0 = 0.f, m1 = -INFINITY, l1 = 0.f;   // running softmax state of the piece
        bool cont_in = false;   // the previous item continues into this one
        for (int u = u0; u < u1; ++u) {
            const int tb = n_tb, te = n_te, nstr = n_nstr, first = n_first, kvh = n_kvh, slot = n_slot;
            const int cut0 = n_cut0, cut1 = n_cut1;
            const bool cont_out = n_cont, sole = kSole && n_sole;
            const int ne = te > tb ? (te - tb + kKT - 1) / kKT : 0, mt = nstr > 16 ? 2 : 1;
            if (u + 1 < u1) fetch_item(u + 1);
            // first partial slot of each row's (stream, KV head), read during the piece's last tile
            int pb0 = 0, pb1 = 0;
            auto fetch_slots = [&]() {
                pb0 = prm.slot_ptr[(size_t)(first + (b0 < nstr ? b0 : 0)) * prm.num_kv_heads + kvh] + slot;
                if (mt == 2) pb1 = prm.slot_ptr[(size_t)(first + (b1 < nstr ? b1 : 0)) * prm.num_kv_heads + kvh] + slot;
            };
            if (!cont_in) {   // a new piece (an item continuing the previous one keeps the state)
                m0 = -INFINITY; l0 = 0.f; m1 = -INFINITY; l1 = 0.f;
            }
            for (int j = 0; j < ne; ++j) {
                if (j == 1 && u + 1 < u1) fetch_cut();
                if (j == ne - 1) fetch_slots();
                // E4M3: for the 16-column blocks 4 hc .. 4 hc + 3 of this thread's column half, the
                // multiplier of the raw scores (log2 units, K scale and 2^112 folded in), the V factor
                // folded into P (as a log2 offset of the exponent) and its inverse for the row sum. A
                // zero scale marks a block without a nonzero value (its codes are zeros): any positive
                // factor gives the same result there.
                float kcb[4], vlb[4], vib[4];
                if constexpr (kE4M3) {
                    const int e = cnt0 % kSclEntries;   // cnt0: tiles so far (every piece has M-tile 0)
                    ok = ok && wait_all(B_SCL + e, (cnt0 / kSclEntries) & 1, 72);
#pragma unroll
                    for (int b = 0; b < 4; ++b) {
                        const float ks = scl[e * 16 + 4 * hc + b], vs = scl[e * 16 + 8 + 4 * hc + b];
                        kcb[b] = c * (ks > 0.f ? ks : 1.f) * kTwo112;
                        const float vf = (vs > 0.f ? vs : 1.f) * kTwo112;
                        vlb[b] = __log2f(vf);
                        vib[b] = fast_exp2(-vlb[b]);
                    }
                }
#pragma unroll
                for (int mi = 0; mi < 2; ++mi) {
                    if (mi >= mt) break;
                    const uint32_t tS = tmem + lanes + 128 * mi, tO = tS + 256;
                    const int cnt = mi ? cnt1 : cnt0;
                    float &m_ref = mi ? m1 : m0;
                    float &l = mi ? l1 : l0;
                    // visible columns of this half: [0, w)
                    const int w = min(max((mi ? cut1 : cut0) - (tb + j * kKT) - 64 * hc, 0), 64);
                    const bool full = __all_sync(0xffffffffu, w == 64);
                    ok = ok && wait_all(B_SFULL + mi, cnt & 1, 70);
                    if (mi) ++cnt1; else ++cnt0;
                    if (!ok) {
                        swap_row(0.f);
                        continue;
                    }
                    tc_fence_after();
                    uint32_t sr[2][32];
                    tmem_ld32(tS + 64 * hc, sr[0]);
                    tmem_ld32(tS + 64 * hc + 32, sr[1]);
                    tmem_ld_wait();
                    if (!full) {
#pragma unroll
                        for (int uu = 0; uu < 2; ++uu) {
                            const uint32_t vis = interval_bits(0, w, uu * 32);
#pragma unroll
                            for (int i = 0; i < 32; ++i) sr[uu][i] = (vis >> i) & 1u ? sr[uu][i] : 0xff800000u;
                        }
                    }
                    float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                    float mx;
                    if constexpr (kE4M3) {
                        // block b = columns 16b .. 16b + 15 of the half: its max, then times its multiplier
#pragma unroll
                        for (int uu = 0; uu < 2; ++uu)
#pragma unroll
                            for (int i = 0; i < 32; i += 4) {
                                const int b = 2 * uu + (i >> 4);
                                mx4[b] = fmax3f(mx4[b], __uint_as_float(sr[uu][i]), __uint_as_float(sr[uu][i + 1]));
                                mx4[b] = fmax3f(mx4[b], __uint_as_float(sr[uu][i + 2]), __uint_as_float(sr[uu][i + 3]));
                            }
                        mx = fmaxf(fmaxf(mx4[0] * kcb[0], mx4[1] * kcb[1]), fmaxf(mx4[2] * kcb[2], mx4[3] * kcb[3]));
                    } else {
#pragma unroll
                        for (int uu = 0; uu < 2; ++uu)
#pragma unroll
                            for (int i = 0; i < 32; i += 8) {
                                mx4[0] = fmax3f(mx4[0], __uint_as_float(sr[uu][i]), __uint_as_float(sr[uu][i + 1]));
                                mx4[1] = fmax3f(mx4[1], __uint_as_float(sr[uu][i + 2]), __uint_as_float(sr[uu][i + 3]));
                                mx4[2] = fmax3f(mx4[2], __uint_as_float(sr[uu][i + 4]), __uint_as_float(sr[uu][i + 5]));
                                mx4[3] = fmax3f(mx4[3], __uint_as_float(sr[uu][i + 6]), __uint_as_float(sr[uu][i + 7]));
                            }
                        mx = fmaxf(fmax3f(mx4[0], mx4[1], mx4[2]), mx4[3]);
                    }
                    // every P store below lands after both halves have read their S columns
                    mx = fmaxf(mx, swap_row(mx));
                    const float m_new = fmaxf(m_ref, mx);
                    // lazy rescaling: the reference max moves only when the row max grew by more
                    // than 2^8 in probability (E4M3: maxima are kept already in log2 units)
                    const bool rescale = m_ref != -INFINITY && (m_new - m_ref) * cm > 8.f;
                    if (m_ref == -INFINITY) m_ref = m_new;
                    float alpha = 1.f;
                    if (rescale) {
                        alpha = fast_exp2((m_ref - m_new) * cm);
                        l *= alpha;
                        m_ref = m_new;
                    }
                    const float moff = m_ref == -INFINITY ? 0.f : m_ref * cm;
                    float rs[4] = {0.f, 0.f, 0.f, 0.f};
                    uint32_t pk[32];
                    if constexpr (kE4M3) {
                        // P of block b carries its V factor (the exponent's log2 offset); rs[b] sums the
                        // block's carried values, and the factor comes off again in the row sum
#pragma unroll
                        for (int qq = 0; qq < 2; ++qq) {
#pragma unroll
                            for (int i = 0; i < 32; i += 2) {
                                const int b = 2 * qq + (i >> 4);
                                const float off = vlb[b] - moff;
                                const float p0 = fast_exp2(fmaf(__uint_as_float(sr[qq][i]), kcb[b], off));
                                const float p1 = fast_exp2(fmaf(__uint_as_float(sr[qq][i + 1]), kcb[b], off));
                                rs[b] += p0 + p1;
                                pk[qq * 16 + (i >> 1)] = pack_bf16x2(p0, p1);
                            }
                        }
                        tmem_st32(tS + 32 * hc, pk);
                        l += (rs[0] * vib[0] + rs[1] * vib[1]) + (rs[2] * vib[2] + rs[3] * vib[3]);
                    } else {
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
                        tmem_st32(tS + 32 * hc, pk);   // P (bf16 pairs) of columns [64 hc, 64 hc + 64)
                        l += (rs[0] + rs[1]) + (rs[2] + rs[3]);
                    }
                    if (__any_sync(0xffffffffu, rescale)) {
                        // PV_i(j-1) completed before S_i(j) (issue order) and PV_i(j) waits for this
                        // warp's P, so O_i is quiescent here
#pragma unroll
                        for (int q = 0; q < 2; ++q) {
                            uint32_t o[32];
                            tmem_ld32(tO + 64 * hc + q * 32, o);
                            tmem_ld_wait();
#pragma unroll
                            for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                            tmem_st32(tO + 64 * hc + q * 32, o);
                        }
                    }
                    tmem_st_wait();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(bar(B_PFULL + mi));
                }
            }
            if (ne < 2 && u + 1 < u1) fetch_cut();
            if (ne == 0) fetch_slots();
            cont_in = cont_out;
            if (cont_out) continue;   // the piece goes on in the next item
            // partials of this piece: O / l (fp32) and the natural-log LSE of every row
#pragma unroll
            for (int mi = 0; mi < 2; ++mi) {
                if (mi >= mt) break;
                const float m_ref = mi ? m1 : m0;
                float l = mi ? l1 : l0;
                if (ne > 0) {
                    ok = ok && wait_all(B_PVDONE + mi, (mi ? pd1 : pd0) & 1, 71);
                    if (mi) ++pd1; else ++pd0;
                }
                l += swap_row(l);   // plus the other column half's sum
                if (!ok) continue;
                tc_fence_after();
                const int b = mi * 16 + row / kGroup;
                const bool valid = b < nstr;
                const bool empty = !(l > 0.f);
                const float inv = empty ? 0.f : 1.f / l;
                const size_t prow = (size_t)(mi ? pb1 : pb0) * kGroup + hl;
                // slot layout [16 chunks of 8 dims][8 heads][8]: the 8 rows (heads) of a stream write
                // one contiguous 256-byte run per chunk; a sole item writes the row's output itself
                __nv_bfloat16 *sb = prm.part_o + (size_t)(mi ? pb1 : pb0) * (kGroup * kD) + hl * 8;
                const size_t orow = ((size_t)(first + (valid ? b : 0)) * prm.num_q_heads + kvh * kGroup + hl);
                __nv_bfloat16 *ob = prm.out + orow * kD + 64 * hc;
                const uint32_t tO = tmem + lanes + 256 + 128 * mi + 64 * hc;
#pragma unroll
                for (int q = 0; q < 2; ++q) {
                    uint32_t o[32];
                    if (ne > 0) {
                        tmem_ld32(tO + q * 32, o);
                        tmem_ld_wait();
                    }
                    if (valid) {
#pragma unroll
                        for (int i = 0; i < 32; i += 8) {
                            auto v = [&](int k) { return empty ? 0.f : __uint_as_float(o[i + k]) * inv; };
                            uint4 w;
                            w.x = pack_bf16x2(v(0), v(1));
                            w.y = pack_bf16x2(v(2), v(3));
                            w.z = pack_bf16x2(v(4), v(5));
                            w.w = pack_bf16x2(v(6), v(7));
                            if (sole) {
                                *reinterpret_cast<uint4 *>(ob + 32 * q + i) = w;
                            } else {
                                const int chunk = 8 * hc + 4 * q + i / 8;
                                *reinterpret_cast<uint4 *>(sb + chunk * (kGroup * 8)) = w;
                            }
                        }
                    }
                }
                if (valid && hc == 0) {
                    const float lv = empty ? -INFINITY : (m_ref * cm + log2f(l)) * PADOC_LN2;
                    if (sole) prm.lse[orow] = lv; else prm.part_lse[prow] = lv;
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

// Registers per thread of the warp path's eight warps (warpgroups 0 and 1) and of warpgroup 2, which
// idles there: 256 x 232 + 128 x 24 = 62,464, within the 384 x 168 = 64,512 the CTA is launched
// with (an increase beyond what the CTA holds would wait forever).
constexpr uint32_t kWarpPathRegs = 232, kIdleRegs = 24;
static_assert(2 * 128 * kWarpPathRegs + 128 * kIdleRegs <= (uint32_t)kThreads * 168, "register split");
static_assert(padoc_warp::kRingBytes <= kSmemBytes && padoc_warp::kRingBytesE4M3 <= kSmemBytes, "warp rings");
static_assert(padoc_warp::kWarps * 32 == 256, "the warp path runs on warpgroups 0 and 1");


// The decode grid (kFused): a CTA runs its tensor-core pieces (CTAs below tc_ctas), then one warp
// CTA's lists on warps 0-7 with the larger register budget (decode_warp.cuh); warps 8-11 give their
// registers back and end. A plan without tensor-core work runs warp CTAs only. Without kFused the
// grid runs the tensor-core pieces only (the E4M3 pool, whose warp lists run in a grid of their own:
// there the warp path needs more registers than the split leaves it). kPreWait: the previous kernel
// in the stream is the step's append (a decoding loop's step), and the warps of CTAs without
// tensor-core pieces start their first paged blocks before they wait for it.
template <bool kE4M3, bool kFused, bool kSole, bool kPreWait>
__global__ void __launch_bounds__(kThreads, 1)
decode_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                 const __grid_constant__ CUtensorMap qmap, const TcDecodeParams prm,
                 const padoc_warp::DecodeParams wprm)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    if (smem_u32(smem) & 1023u) {
        if (threadIdx.x == 0) padoc_record_error(prm.err, PADOC_DEVERR_SMEM_ALIGN, (int)(smem_u32(smem) & 1023u));
        return;
    }
    const bool has_tc = (int)blockIdx.x < prm.tc_ctas;
    if constexpr (!kFused) {
        if (has_tc) decode_tc_role<kE4M3, false, kSole>(kmap, vmap, qmap, prm, wprm, smem);
        return;
    }
    if (has_tc) {
        decode_tc_role<kE4M3, true, kSole>(kmap, vmap, qmap, prm, wprm, smem);
    } else if constexpr (!kPreWait) {
        // a CTA with warp lists only: the same wait for the previous kernel in the stream (kPreWait:
        // each warp of the warp path waits itself, after its first loads)
        pdl_wait_prerequisite();
        pdl_launch_dependents();
    }
    const int wc = has_tc ? prm.early_ctas + (int)blockIdx.x : (int)blockIdx.x - prm.tc_ctas;
    const bool lists = wc < prm.warp_ctas;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp >= padoc_warp::kWarps) {
        if (lists) setmaxnreg_dec<kIdleRegs>();
        return;
    }
    if (!lists) return;
    setmaxnreg_inc<kWarpPathRegs>();
    // the rings reuse shared memory that the tensor cores and TMA (the async proxy) last accessed
    fence_proxy_async_smem();
    const int wi = wc * padoc_warp::kWarps + warp;
    if (wi >= wprm.num_warps) return;
    if (kPreWait && !has_tc)
        padoc_warp::decode_warp_role<kE4M3, true>(wprm, smem, warp, lane, wi);
    else
        padoc_warp::decode_warp_role<kE4M3, false>(wprm, smem, warp, lane, wi);
}

}  // namespace

padoc_status padoc_launch_decode_tc(const CUtensorMap *kmap, const CUtensorMap *vmap, const CUtensorMap *qmap, const int32_t *plan,
                                    const padoc_decode_plan *info, const int32_t *page_table, int32_t page_stride,
                                    const int32_t *stream_table, int32_t stream_stride, int32_t num_blocks,
                                    const float *k_scales, const float *v_scales, __nv_bfloat16 *part_o, float *part_lse,
                                    __nv_bfloat16 *out, float *lse, float scale_log2, int *err,
                                    const padoc_warp::DecodeParams *wprm, cudaStream_t stream)
{
    const bool e4m3 = k_scales != nullptr;   // an E4M3 pool: the maps hold codes
    const bool fused = !e4m3;
    if (info->num_tc_items == 0 && (!fused || wprm->num_warps == 0)) return PADOC_OK;
    TcDecodeParams prm;
    prm.shared_len = plan + info->off_shared_len;
    prm.private_len = plan + info->off_private_len;
    prm.slot_ptr = plan + info->off_slot_ptr;
    prm.cta_ptr = plan + info->off_cta_ptr;
    prm.items = reinterpret_cast<const padoc_item *>(plan + info->off_items);
    prm.num_tc_items = info->num_tc_items;
    prm.num_pages = info->num_pages;
    prm.num_streams = info->num_streams;
    prm.page_table = page_table;
    prm.page_stride = page_stride;
    prm.stream_table = stream_table;
    prm.stream_stride = stream_stride;
    prm.num_blocks = num_blocks;
    prm.num_kv_heads = info->cfg.num_kv_heads;
    prm.pool_rows = num_blocks * info->cfg.num_kv_heads * kBlk;
    prm.k_scales = k_scales;
    prm.v_scales = v_scales;
    prm.part_o = part_o;
    prm.part_lse = part_lse;
    prm.out = out;
    prm.lse = lse;
    prm.num_q_heads = info->cfg.num_q_heads;
    prm.scale_log2 = scale_log2;
    prm.err = err;
    prm.tc_ctas = info->num_tc_items > 0 ? info->tc_ctas : 0;
    prm.warp_ctas = fused ? (wprm->num_warps + padoc_warp::kWarps - 1) / padoc_warp::kWarps : 0;
    prm.early_ctas = padoc_fused_early_ctas(prm.tc_ctas, prm.warp_ctas, padoc_default_ctas());
    // plans with sole items (chunked prefill) take the variant that writes their outputs
    const bool sole = (int64_t)info->num_merge_keys < (int64_t)info->num_streams * info->cfg.num_kv_heads;
    // a decoding-loop step right after its append (no sole items): warps of warp-only CTAs load
    // before they wait
    const bool pre_wait = fused && wprm->pre_wait && !sole;
    auto kern = e4m3       ? (sole ? decode_tc_kernel<true, false, true, false> : decode_tc_kernel<true, false, false, false>)
                : pre_wait ? decode_tc_kernel<false, true, false, true>
                           : (sole ? decode_tc_kernel<false, true, true, false> : decode_tc_kernel<false, true, false, false>);
    {
        const padoc_status ast = padoc_set_max_smem(reinterpret_cast<const void *>(kern), (int)kSmemBytes);
        if (ast != PADOC_OK) return ast;
    }
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3((unsigned)(prm.tc_ctas + prm.early_ctas));
    lc.blockDim = dim3(kThreads);
    lc.dynamicSmemBytes = kSmemBytes;
    lc.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // see the kernel's wait
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = 1;
    PADOC_CUDA_TRY(cudaLaunchKernelEx(&lc, kern, *kmap, *vmap, *qmap, prm, *wprm));
    return padoc_launch_status();
}
