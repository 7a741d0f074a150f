// plan_internal.h -- layouts shared by the host planner and the CUDA kernels of padoc_attn.
#pragma once

#include <stddef.h>
#include <stdint.h>

// Prefill tiles: 128 query rows x 128 key columns (one tcgen05 M=128 tile by N=128 keys; the
// warp-MMA kernel walks the same tile map).
#define PADOC_PREFILL_Q_TILE 128
#define PADOC_PREFILL_K_TILE 128

// Decode split-K: shared-stream tokens per partial result, private tokens per partial result, and
// streams (8 query heads each) per warp-MMA work item.
#define PADOC_DEFAULT_SPLIT_TOKENS 512
#define PADOC_PRIVATE_SPLIT_TOKENS 512
#define PADOC_MMA_ROW_STREAMS 4

#define PADOC_ITEM_INTS 8
enum { PADOC_ITEM_SHARED = 0, PADOC_ITEM_PRIVATE = 1 };

// One split-K work item of the decode kernels (8 int32 words in the plan blob).
//   kind        PADOC_ITEM_SHARED: tokens [tok_begin, tok_end) of page `index`'s shared stream for
//               streams [first_stream, first_stream + num_streams) of that page, each with its own
//               column cutoff shared_len;
//               PADOC_ITEM_PRIVATE: private tokens [tok_begin, tok_end) of stream `index`.
//   kv_head     the KV head; the item covers that head's Hq/Hkv query heads of every stream.
//   slot        partial-result slot of each covered stream s: slot_ptr[s] + slot.
typedef struct {
    int32_t kind, index, kv_head, tok_begin, tok_end, first_stream, num_streams, slot;
} padoc_item;

static inline size_t padoc_align256(size_t x) { return (x + 255) & ~(size_t)255; }

// Workspace: part_o fp32 [slots][Hq][d], then part_lse fp32 [slots][Hq] at a 256-byte boundary.
static inline size_t padoc_decode_workspace_bytes(int64_t slots, int32_t hq, int32_t d)
{
    return padoc_align256((size_t)slots * hq * d * 4) + padoc_align256((size_t)slots * hq * 4);
}
