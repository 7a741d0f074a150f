// plan_build.h -- host-only internals of the decode planner (plan.cpp), shared with the decoding
// loop's scheduler (mpd.cpp), which plans each step from its stream list in one pass.
#pragma once

#include <stdint.h>

#include <vector>

#include "padoc_attn.h"
#include "plan_internal.h"

struct PlanStream { int32_t page, shared_len, private_len; };

// One (KV head, page, group of streams) of tensor-core work and the shared-stream tiles it sees, with
// the private continuation of a chunked prefill's group (ntiles2 = 0: none); build_work's comment has
// the rest.
struct PlanSegment {
    int32_t kind, g, p, first, ns, vis, ntiles, weight;
    int32_t kind2, p2, vis2, ntiles2;
};

// Working arrays of build_work, kept with the parts so that a caller planning step after step (the
// decoding loop's scheduler) reuses their memory.
struct PlanScratch {
    std::vector<uint8_t> priv_tc, direct;
    std::vector<int32_t> cnt, perm, ptr_sorted, cost, order, counts, nw_of, by_start, head, tail, next, warp_of, wpos;
    std::vector<int64_t> tc_load, load_sorted, room;
    std::vector<double> start, rate, tend;
    std::vector<padoc_item> tc_items, items_sorted, warp_items;
    std::vector<PlanSegment> segs;
    // the tensor-core bound search's inputs (want, chunked, each segment's tiles and weight) and its
    // result, from the last search (bound < 0: none yet)
    std::vector<int64_t> bound_key, last_bound_key;
    int64_t bound = -1;
};

struct PlanParts {
    std::vector<PlanStream> streams;
    std::vector<int32_t> page_len, page_first_stream, page_num_streams;
    std::vector<int32_t> slot_ptr;      // [S * Hkv + 1]: partial slots of each (stream, KV head)
    std::vector<int32_t> cta_ptr;       // [tc_ctas + 1]: tensor-core items of each CTA
    std::vector<int32_t> warp_ptr;      // [num_warps + 1]: warp items of each warp (from the first)
    std::vector<int32_t> merge_keys;    // the (stream, KV head) keys the merge joins (the others are written directly)
    std::vector<padoc_item> items;
    int32_t num_tc_items = 0, tc_ctas = 0, num_warps = 0;
    int32_t tc_min_rows = PADOC_TC_MIN_ROWS;   // rows from which a page's shared stream goes to the tensor cores
    int32_t max_page_blocks = 0, max_stream_blocks = 0;
    int64_t kv_tokens = 0;
    // chunked prefill plans only (empty otherwise): the chunk of each stream, and per chunk its
    // first stream, its token count and whether its tokens have private rows
    std::vector<int32_t> chunk_of, chunk_first, chunk_len;
    std::vector<uint8_t> chunk_private;
    PlanScratch scratch;

    // Empties every part (their memory and the scratch arrays stay allocated).
    void reset()
    {
        streams.clear();
        page_len.clear();
        page_first_stream.clear();
        page_num_streams.clear();
        slot_ptr.clear();
        cta_ptr.clear();
        warp_ptr.clear();
        merge_keys.clear();
        items.clear();
        num_tc_items = tc_ctas = num_warps = 0;
        tc_min_rows = PADOC_TC_MIN_ROWS;
        max_page_blocks = max_stream_blocks = 0;
        kv_tokens = 0;
        chunk_of.clear();
        chunk_first.clear();
        chunk_len.clear();
        chunk_private.clear();
    }
};

// The split-K work of an explicit stream list (padoc_build_decode_plan_streams' rules).
padoc_status padoc_plan_parts_of_list(const int32_t *page_len, int32_t num_pages, const padoc_stream_desc *streams,
                                      int32_t num_streams, const padoc_decode_config *cfg, PlanParts &pp);
// The streams of a chunked prefill (padoc_build_chunk_prefill_plan's rules) and their work.
padoc_status padoc_plan_parts_of_chunks(const int32_t *page_len, int32_t num_pages, const padoc_prefill_chunk *chunks,
                                        int32_t num_chunks, const padoc_decode_config *cfg, PlanParts &pp);
// int32 words of the plan blob of pp.
int64_t padoc_plan_blob_ints(const PlanParts &pp, int32_t num_pages, int32_t hkv);
// Writes the blob and its host summary (CAPACITY when capacity_ints is too small).
padoc_status padoc_plan_write_blob(const PlanParts &pp, int32_t num_pages, const padoc_decode_config *cfg, int32_t *plan,
                                   int64_t capacity_ints, padoc_decode_plan *info);

// padoc_branch_decode_attn for a decoding-loop step launched right after that step's append on the
// same stream (padoc_mpd_launch_step): the append writes only each stream's newest K/V row and the
// step's queries, and the plan and block tables were copied before it started, so warps without
// tensor-core work read those and start their first paged blocks before they wait for the append.
// first_blocks (device, may be NULL): int32 [num_warps][4], the pool rows of the first four blocks
// of each warp's first item (-2 - row for the block of its stream's newest row, -1 past its end),
// read in parallel with the item headers (padoc_mpd_step.off_first_blocks).
padoc_status padoc_branch_decode_attn_after_append(const padoc_kv_pool *pool, const padoc_decode_plan *info,
                                                   const int32_t *plan_dev, const int32_t *page_block_table,
                                                   int32_t page_table_stride, const int32_t *stream_block_table,
                                                   int32_t stream_table_stride, const void *q, float scale, void *out,
                                                   float *lse, void *workspace, size_t workspace_bytes,
                                                   padoc_stream_t stream, const int32_t *first_blocks);
