// plan_internal.h -- layouts shared by the host planner and the CUDA kernels of padoc_attn.
#pragma once

#include <stddef.h>
#include <stdint.h>

// Prefill tiles: 128 query rows x 128 key columns (one tcgen05 M = 128 tile by N = 128 keys).
#define PADOC_PREFILL_Q_TILE 128
#define PADOC_PREFILL_K_TILE 128

// Prefill backward tiles. The dQ pass keeps 128 query rows (the M of its MMAs) and walks 64-key
// k-tiles; the dK/dV pass keeps 128 keys (the M of its MMAs) and walks 64-row q-tiles. Narrow
// steps let two steps' scores sit in tensor memory beside the accumulators and the resident A
// operands, so the exponentials of one step overlap the MMAs of the next one (128-key dQ steps, one
// step buffer, halve the S and dP MMA instructions but serialize the two: 1.305 -> 1.388 ms).
#define PADOC_BWD_DQ_Q_TILE 128
#ifndef PADOC_BWD_DQ_K_TILE
#define PADOC_BWD_DQ_K_TILE 64
#endif
#define PADOC_BWD_DKV_Q_TILE 64
#define PADOC_BWD_DKV_K_TILE 128
// A dK/dV work unit (k-tile, KV head) of more steps ((q-tile, query head) pairs) than this is split
// between two CTAs, each over half of its steps, whose fp32 partials a small kernel adds: the first
// k-tiles of a page are seen by up to 64 q-tiles x 8 heads, and as single CTAs they set the pass's
// tail (measured: 927 us against 681 us of work per SM). Only the heaviest units can split (those
// whose position in the key-major order is below k-tiles / KV heads), so that the partials fit in
// PADOC_BWD_SPLIT_BYTES_PER_TOKEN bytes of workspace per token.
#define PADOC_BWD_SPLIT_STEPS 256
#define PADOC_BWD_SPLIT_BYTES_PER_TOKEN 2048

// Decode split-K: shared-stream tokens per partial result and private tokens per partial result.
// 256 rather than 512: in decoding-loop steps with few streams the warp items on a page's shared
// stream are the critical path (measured on GB300: 31 -> 21 us per step at 1-2 live streams), and
// the one-shot serving batch, whose shared streams go to the tensor cores, does not change.
#define PADOC_DEFAULT_SPLIT_TOKENS 256
// Longest warp item: a warp keeps one block id per lane, so an item spans at most 32 blocks.
#define PADOC_WARP_MAX_ITEM_TOKENS 512
#define PADOC_PRIVATE_SPLIT_TOKENS 256
// The planner's own split (split_tokens 0) is 64 tokens below this many 16-token blocks of warp work
// per warp of the grid and 128 below the next; 256 above.
#ifndef PADOC_SPLIT_64_BLOCKS
#define PADOC_SPLIT_64_BLOCKS 3
#endif
#ifndef PADOC_SPLIT_128_BLOCKS
#define PADOC_SPLIT_128_BLOCKS 8
#endif
// Shared-stream rows (streams x query heads of one KV head) from which the tensor-core kernel
// takes a page: below this the rows are too few for a dense M = 128 contraction and each stream
// reads the shared stream with warp-level MMAs instead.
#ifndef PADOC_TC_MIN_ROWS
#define PADOC_TC_MIN_ROWS 64
#endif
// ... and from this many in a decode plan with much warp work (at least PADOC_TC_BUSY_BLOCKS
// 16-token blocks per warp of the grid): two streams of eight query heads
#ifndef PADOC_TC_MIN_ROWS_BUSY
#define PADOC_TC_MIN_ROWS_BUSY 16
#endif
#ifndef PADOC_TC_BUSY_BLOCKS
#define PADOC_TC_BUSY_BLOCKS 6
#endif
// Streams per tensor-core work item: two M = 128 tiles of 16 streams x 8 query heads.
#define PADOC_TC_ITEM_STREAMS 32
// Tokens per K/V tile of the tensor-core kernel, and the relative cost of one tile for a group of
// more than 16 streams (two M-tiles) and of at most 16 (one M-tile), used to balance CTAs.
#define PADOC_TC_TILE_TOKENS 128
#define PADOC_TC_WEIGHT_2M 8
#define PADOC_TC_WEIGHT_1M 7
// Fixed cost of one tensor-core piece in the same units (its partials' epilogue and the reload of
// the queries before it), fitted on GB300 to per-CTA timelines of the serving batch: about one tile
// for a one-M-tile piece, a tile and a half for a two-M-tile piece
#define PADOC_TC_PIECE_COST_1M 7
#define PADOC_TC_PIECE_COST_2M 11
// ... plus this for a piece of a chunked prefill (a group's shared tiles and then its private ones:
// two items, the switch between them, and tiles that other groups read too), fitted to per-CTA
// timelines of the serving batch's branch prefill
#ifndef PADOC_TC_PIECE_EXTRA_CHUNK
#define PADOC_TC_PIECE_EXTRA_CHUNK 15
#endif

// Warps per CTA of the warp kernel, and the start-up cost of one warp item in 16-token blocks
// (query fragments, the first blocks' latency, the partial's write), used to balance warps.
#define PADOC_WARP_KERNEL_WARPS 8
#define PADOC_WARP_ITEM_COST 2
// Timing model of one decode step, fitted on GB300 to per-CTA and per-warp timelines of the serving
// batch (times in microseconds from the start of the decode grid), used to size each warp's share:
// a tensor-core CTA with a planned load of L units (the weights above) ends at about
// PADOC_TC_END_US0 + PADOC_TC_US_PER_UNIT * L; a warp CTA on an SM the tensor-core CTAs leave free
// starts at PADOC_WARP_EARLY_START_US and works through PADOC_WARP_EARLY_RATE cost units (16-token
// blocks plus PADOC_WARP_ITEM_COST per item) per microsecond; one that a tensor-core CTA runs after
// its pieces starts PADOC_WARP_SWITCH_US after they end, needs PADOC_WARP_FIRST_US before its first
// block lands (the memory system is busiest then) and then works through PADOC_WARP_RATE units per
// microsecond.
#ifndef PADOC_TC_END_US0
#define PADOC_TC_END_US0 5.6
#endif
#ifndef PADOC_TC_US_PER_UNIT
#define PADOC_TC_US_PER_UNIT 0.238
#endif
// the last tensor-core CTA of a step ends about this long after the average one
#ifndef PADOC_TC_END_SPREAD_US
#define PADOC_TC_END_SPREAD_US 2.5
#endif
#ifndef PADOC_WARP_EARLY_START_US
#define PADOC_WARP_EARLY_START_US 5.2
#endif
#ifndef PADOC_WARP_SWITCH_US
#define PADOC_WARP_SWITCH_US 0.2
#endif
#ifndef PADOC_WARP_FIRST_US
#define PADOC_WARP_FIRST_US 5.3
#endif
#ifndef PADOC_WARP_RATE
#define PADOC_WARP_RATE 1.53
#endif
#ifndef PADOC_WARP_EARLY_RATE
#define PADOC_WARP_EARLY_RATE 1.28
#endif

// The fused decode grid: CTA c < tc_ctas runs tensor-core CTA c's pieces and then one warp CTA's
// lists (8 warps); the CTAs from tc_ctas on run warp CTAs' lists from the start. Warp CTAs
// [0, early) go to CTAs tc_ctas + c (the SMs the tensor-core CTAs leave free: they start first, so
// the planner gives them the longest items), warp CTA early + j to tensor-core CTA j. early is the
// number of free SMs, raised where needed so that every warp CTA has a CTA:
// max(min(warp_ctas, sm_count - tc_ctas), warp_ctas - tc_ctas, 0). The grid has tc_ctas + early CTAs.
static inline int32_t padoc_fused_early_ctas(int32_t tc_ctas, int32_t warp_ctas, int32_t sm_count)
{
    int32_t e = sm_count - tc_ctas;
    if (e > warp_ctas) e = warp_ctas;
    if (e < warp_ctas - tc_ctas) e = warp_ctas - tc_ctas;
    return e > 0 ? e : 0;
}

#define PADOC_ITEM_INTS 8
enum { PADOC_ITEM_SHARED = 0, PADOC_ITEM_PRIVATE = 1, PADOC_ITEM_SHARED_TC = 2, PADOC_ITEM_PRIVATE_TC = 3 };
// Flag added to the kind of a tensor-core item of a chunked prefill whose rows other groups read
// too (a page with more than 32 chunk tokens, a chunk of more than 32 tokens): its tiles are loaded
// with the normal L2 policy so that the groups running at the same time share them. Decode plans
// never set it: their tiles are loaded evict-first, which keeps the split-K partials in L2 for the
// merge (measured: flagging the decode step's pages of more than 32 streams was no faster).
#define PADOC_ITEM_REREAD 16
// Flag of a tensor-core item that the next item of the same CTA continues (a chunked prefill's
// piece over a group's shared tiles and then its private ones): the same streams, KV head and
// partial slot, one running softmax over both, one partial written after the second item.
#define PADOC_ITEM_CONT 32
// Flag of a tensor-core item that is the only partial of each of its streams for its KV head: it
// writes their bf16 outputs and LSE itself (exactly the merge's result for one partial), and the
// merge skips those keys (a chunked prefill's groups whose pieces stay on one CTA).
#define PADOC_ITEM_SOLE 64
#define PADOC_ITEM_KIND(k) ((k) & 15)

// One split-K work item of the decode kernels (8 int32 words in the plan blob). The blob holds
// the tensor-core items first ([0, num_tc_items)), tensor-core CTA c owning items
// [cta_ptr[c], cta_ptr[c+1]) in order, then the warp items, warp w (warp w % 8 of warp CTA w / 8)
// owning items num_tc_items + [warp_ptr[w], warp_ptr[w+1]) in order. A warp item's tok_end never passes
// its stream's cutoff (shared_len or private_len), so the warp kernel reads no cutoff.
//   kind        PADOC_ITEM_SHARED_TC: tokens [tok_begin, tok_end) of page `index`'s shared stream for
//               streams [first_stream, first_stream + num_streams) (<= 32) of that page, each with
//               its own column cutoff shared_len (tensor-core kernel);
//               PADOC_ITEM_SHARED: the same for the one stream first_stream (warp kernel);
//               PADOC_ITEM_PRIVATE: private tokens [tok_begin, tok_end) of stream `index` (warp kernel);
//               PADOC_ITEM_PRIVATE_TC: private tokens [tok_begin, tok_end) of a chunk of consecutive query
//               tokens of one stream: streams [first_stream, first_stream + num_streams) (<= 32), each
//               with its own cutoff private_len, all reading the private block-table row of stream
//               `index`, the chunk's first token (tensor-core kernel).
//   kv_head     the KV head; the item covers that head's Hq/Hkv query heads of every stream.
//   slot        partial-result slot of each covered stream s: slot_ptr[s * Hkv + kv_head] + slot.
typedef struct {
    int32_t kind, index, kv_head, tok_begin, tok_end, first_stream, num_streams, slot;
} padoc_item;

static inline size_t padoc_align256(size_t x) { return (x + 255) & ~(size_t)255; }

// Workspace: part_o bf16 [slots][d / 8][group][8] (a slot's dims in chunks of 8, the group's heads
// inside a chunk, so that the heads of one stream are written as one contiguous run per chunk; each
// partial is O / l, so bf16 adds at most 2^-9 of its magnitude before the merge's fp32 sums), then
// part_lse fp32 [slots][group] at a 256-byte boundary; a slot holds one partial of the
// group = Hq / Hkv query heads of one (stream, KV head).
static inline size_t padoc_decode_workspace_bytes(int64_t slots, int32_t group, int32_t d)
{
    return padoc_align256((size_t)slots * group * d * 2) + padoc_align256((size_t)slots * group * 4);
}
