/*
 * padoc_attn.h -- C ABI of padoc_attn, ancestor-masked attention over one shared page
 * representation for PaDoc's layout-grounded parallel decoding, on one NVIDIA GB300 (sm_103a).
 *
 * The visibility rule (Sec. 3.2, ancestor sets Anc(B_k) = {X, B_<k}, Anc(Y_k) = {X, B_<=k};
 * App. C.1, Q_M -> K_M causal and Q_{Y_k} -> [K_{M<=f_k}; K_{Y_k}] with bottom-right causality;
 * App. E.1, the additive-bias softmax and Algorithm 1). A page is packed as
 *
 *     [ prefix X (P tokens) | layout stream (L tokens) | Y_1 (n_1) | ... | Y_N (n_N) ]
 *
 * and a token at page-local position q may see page-local key j exactly when
 *     q < P + L          :  j <= q                                   (one causal stream)
 *     q = ybase_k + i    :  j < P + f_k   or   ybase_k <= j <= q     (two spans)
 * Tokens of different pages never see each other. f_k (0 <= f_k <= L) is the number of
 * layout-stream tokens visible to branch k: Algorithm 1 forks a branch with a copy of the layout
 * stream's row taken before the region's boundary output is appended. Any order of f_k and ties
 * are legal (one branch-start token per extra branch at a higher-arity fork, Sec. 3.2).
 *
 * For each query and query head h, with KV head g = h / (Hq / Hkv):
 *     s_j = scale * q . k_j (visible j),  lse = ln sum_j exp(s_j),  o = sum_j exp(s_j - lse) v_j.
 *
 * Conventions for every call
 *   - Ownership: the caller owns every buffer. The library never allocates device memory, never
 *     keeps a pointer after a call returns and never synchronizes, except
 *     padoc_check_device_errors. The objects it allocates are the decoding loop's host-side
 *     scheduler state (padoc_mpd_create / padoc_mpd_destroy) and the loop's step runner
 *     (padoc_mpd_runner_*), which owns its staging and device buffers, keeps the scheduler and pool
 *     it was made for, and waits for its own events.
 *   - Host pointers are marked (host); device pointers (device). Device calls are asynchronous on
 *     the given stream (a cudaStream_t; NULL is the legacy default stream).
 *   - Every argument is validated on the host before any launch; a failed check returns
 *     PADOC_ERR_INVALID_ARGUMENT (or _UNSUPPORTED / _WORKSPACE_TOO_SMALL / _CAPACITY) and launches
 *     nothing. There is no fallback path: an unsupported combination is an error.
 *   - Block ids read on the device are range-checked; a bad id sets a device error word (read with
 *     padoc_check_device_errors), the block is not read, and the call's outputs are undefined.
 *   - Every wait inside a kernel is bounded; a wait that runs out sets the device error word and
 *     the kernel returns.
 *   - Query heads map to KV heads in consecutive groups: h -> h / (Hq / Hkv).
 *   - LSE is the natural-log log-sum-exp, fp32, laid out [query][head].
 */
#ifndef PADOC_ATTN_H
#define PADOC_ATTN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* 1: descriptors, decode, prefill, combine, prefill backward, no-alloc decode. 2 adds the
 * stream-list and chunked-prefill planners, Algorithm 1's loop (padoc_mpd_*) and the append call.
 * 3 adds the FP8 (E4M3) KV cache (padoc_kv_pool_e4m3 and its quantize, append and decode calls),
 * the bounded-wait self-test, the in-place plan advance and the one-call decode step. 4 adds the
 * merge key list to the decode plan (padoc_decode_plan.off_merge_keys, num_merge_keys). 5 adds the
 * loop's step runner (padoc_mpd_runner_*). 6 adds padoc_mpd_step.off_first_blocks and stores the
 * split-K partials in bf16 (the decode workspace's size changes with it). */
#define PADOC_ATTN_VERSION 6

/* A CUDA stream handle; identical to cudaStream_t. */
typedef struct CUstream_st *padoc_stream_t;
/* A CUDA event handle; identical to cudaEvent_t. */
typedef struct CUevent_st *padoc_event_t;

typedef enum {
    PADOC_OK = 0,
    PADOC_ERR_INVALID_ARGUMENT = 1,    /* a size, range, pointer or layout check failed */
    PADOC_ERR_UNSUPPORTED = 2,         /* valid, but not a combination this build implements */
    PADOC_ERR_WORKSPACE_TOO_SMALL = 3, /* workspace_bytes below padoc_decode_workspace_size */
    PADOC_ERR_CUDA = 4,                /* a CUDA runtime call or launch failed */
    PADOC_ERR_DEVICE_CHECK = 5,        /* a kernel reported a failed device-side check */
    PADOC_ERR_CAPACITY = 6             /* a caller-sized output array is too small */
} padoc_status;

typedef enum { PADOC_DTYPE_F32 = 0, PADOC_DTYPE_BF16 = 1 } padoc_dtype;

/* Tile classes of the prefill tile map. */
enum { PADOC_TILE_PARTIAL = 1, PADOC_TILE_FULL = 2 };

/* One page (host). Sec. 3.2 / App. C.1.
 *   prefix_len   P >= 0: image and prompt tokens (the node X), causal inside.
 *   layout_len   L >= 0: layout-stream tokens (B_1..B_N serialized), causal, sees all of X.
 *   num_branches N >= 0.
 *   fork_offset  [N], 0 <= f_k <= L: layout tokens visible to branch k.
 *   branch_len   [N], >= 1: prefill: tokens of Y_k (its branch-start token included);
 *                decode: private KV length of branch k, including the token being decoded
 *                (Algorithm 1 appends every live stream's input before it decodes).
 * A page must hold at least one token. */
typedef struct {
    int32_t prefix_len;
    int32_t layout_len;
    int32_t num_branches;
    const int32_t *fork_offset;
    const int32_t *branch_len;
} padoc_page;

/* ============================================================================================
 * C1: ancestor descriptors (host, integer only, bit-exact; caller-allocated outputs)
 * ========================================================================================== */

/* Total packed tokens T = sum over pages of P + L + sum_k n_k (must be < 2^31).
 * Errors: INVALID_ARGUMENT for a null pointer or a malformed page. */
padoc_status padoc_packed_size(const padoc_page *pages, int32_t num_pages, int64_t *total_tokens);

/* Per-query visible spans (App. C.1 packed relation), absolute packed indices (pages packed
 * back to back in the given order):
 *   spans[4t+0], spans[4t+1] : first span  [kv0_begin, kv0_end)
 *   spans[4t+2], spans[4t+3] : second span [kv1_begin, kv1_end)
 * Prefix/layout token q of a page starting at pb: first = [pb, q+1), second empty.
 * Branch token q of Y_k: first = [pb, pb+P+f_k), second = [ybase_k, q+1).
 * An empty second span is written {kv0_end, kv0_end}. spans: (host) int32 [capacity_tokens][4].
 * Errors: INVALID_ARGUMENT; CAPACITY when capacity_tokens < T. */
padoc_status padoc_build_query_spans(const padoc_page *pages, int32_t num_pages, int32_t *spans,
                                     int64_t capacity_tokens);

/* Tile shape (q_tile, k_tile) the prefill kernel for (dtype, head_dim) consumes. */
padoc_status padoc_prefill_tile_shape(padoc_dtype dtype, int32_t head_dim, int32_t *q_tile, int32_t *k_tile);

/* Size of the prefill tile map for tiles of q_tile query rows by k_tile key columns:
 * num_q_tiles = ceil(T / q_tile); nnz = number of (q-tile, k-tile) pairs with a visible entry. */
padoc_status padoc_tile_map_size(const padoc_page *pages, int32_t num_pages, int32_t q_tile, int32_t k_tile,
                                 int64_t *num_q_tiles, int64_t *nnz);

/* Prefill work list in CSR form (Flex-Attention-style block skipping, App. C.1): for q-tile r,
 * entries [row_ptr[r], row_ptr[r+1]) list the k-tiles holding at least one visible
 * (query, key) pair, in ascending k-tile order, with kinds[e] = PADOC_TILE_FULL when every query
 * row of the tile that exists (< T) sees all k_tile columns (a k-tile reaching past T is never
 * FULL) and PADOC_TILE_PARTIAL otherwise. Fully masked tiles are absent.
 * row_ptr: (host) int32 [num_q_tiles + 1]; k_tiles: (host) int32 [capacity_nnz];
 * kinds: (host) int8 [capacity_nnz]. Errors: INVALID_ARGUMENT; CAPACITY when capacity_nnz < nnz. */
padoc_status padoc_build_tile_map(const padoc_page *pages, int32_t num_pages, int32_t q_tile, int32_t k_tile,
                                  int32_t *row_ptr, int32_t *k_tiles, int8_t *kinds, int64_t capacity_nnz);

/* Key-major (CSC) form of the same work list, for the dK/dV pass of the prefill backward, where
 * every key's gradient sums over all queries that see it (App. C.1: the backward of the
 * tree-varlen gather scatter-adds onto the shared rows). For k-tile c, entries
 * [col_ptr[c], col_ptr[c+1]) list the q-tiles holding a visible pair in ascending order, with the
 * kinds padoc_build_tile_map gives the same (q-tile, k-tile) pair. k_order lists every k-tile once,
 * those with more entries first (ties in ascending order): the order the dK/dV pass takes them.
 * col_ptr: (host) int32 [ceil(T / k_tile) + 1]; q_tiles: (host) int32 [capacity_nnz];
 * kinds: (host) int8 [capacity_nnz]; k_order: (host) int32 [ceil(T / k_tile)].
 * nnz is the one padoc_tile_map_size reports. Errors: INVALID_ARGUMENT; CAPACITY. */
padoc_status padoc_build_key_tile_map(const padoc_page *pages, int32_t num_pages, int32_t q_tile, int32_t k_tile,
                                      int32_t *col_ptr, int32_t *q_tiles, int8_t *kinds, int32_t *k_order,
                                      int64_t capacity_nnz);

/* Tile shapes the prefill backward for (dtype, head_dim) consumes: the dQ pass reads a query-major
 * map (padoc_build_tile_map) of dq_q_tile x dq_k_tile tiles, the dK/dV pass a key-major map
 * (padoc_build_key_tile_map) of dkv_q_tile x dkv_k_tile tiles. Errors: INVALID_ARGUMENT,
 * UNSUPPORTED. */
padoc_status padoc_prefill_bwd_tile_shapes(padoc_dtype dtype, int32_t head_dim, int32_t *dq_q_tile,
                                           int32_t *dq_k_tile, int32_t *dkv_q_tile, int32_t *dkv_k_tile);

/* ============================================================================================
 * C5 + C2 + C4: paged KV cache and one decode step for every live stream (App. E.1, Alg. 1)
 * ========================================================================================== */

/* The paged KV pool (device), C5. Blocks of block_size tokens; per block, per KV head, the
 * block_size x head_dim rows are contiguous: k_pool/v_pool are [num_blocks][num_kv_heads]
 * [block_size][head_dim] in dtype, 16-byte aligned. A page's shared stream (prefix + layout, the
 * tokens every branch of the page shares) is stored once, addressed by the page's block table;
 * each stream's private tokens live in its own blocks starting at block offset 0, addressed by
 * the stream's block table. Visibility is a per-stream column cutoff, so nothing is duplicated
 * (the paper's serving reuses only complete shared blocks and re-prefills the tail, App. E.2). */
typedef struct {
    const void *k_pool;
    const void *v_pool;
    int32_t num_blocks;
    int32_t block_size;   /* 16 */
    int32_t num_kv_heads;
    int32_t head_dim;     /* 128 (bf16) or 64/128 (f32) */
    padoc_dtype dtype;
} padoc_kv_pool;

typedef struct {
    int32_t num_q_heads;
    int32_t num_kv_heads;
    int32_t head_dim;
    int32_t block_size;      /* must equal the pool's block_size */
    int32_t layout_streams;  /* 1: also decode each page's layout stream (Alg. 1 decodes every live
                                stream): cutoff P + L over the shared stream, no private rows */
    int32_t split_tokens;    /* shared-stream tokens per split-K partial of the warp kernel (pages with
                                too few streams for the tensor cores); a positive value must be a
                                multiple of block_size, values above 512 act as 512, and private
                                histories are then cut every 256 tokens; 0 = the planner's choice:
                                256 tokens for both, or 128 / 64 when the warp work is small
                                against the warp grid (a decoding loop's steps with few streams) */
    int32_t tc_ctas;         /* CTAs the tensor-core shared-stream work is balanced over (one range of
                                equal work each); 0 = the current device's multiprocessor count */
    int32_t warp_ctas;       /* CTAs (of 8 warps) the warp-kernel work is balanced over, one wave;
                                0 = the current device's multiprocessor count */
} padoc_decode_config;

/* Host summary of a decode plan, filled by padoc_build_decode_plan. The int32 plan blob it
 * describes must be copied to the device unchanged and passed as plan_dev.
 * Streams are ordered page by page: the page's branches in the given order, then (with
 * layout_streams) its layout stream. Q, out and lse rows follow this order. */
typedef struct {
    padoc_decode_config cfg;
    int32_t num_pages;
    int32_t num_streams;
    int32_t num_items;         /* work items of the split-K decode kernels */
    int32_t num_tc_items;      /* of which use the tensor-core shared-stream kernel */
    int32_t tc_ctas;           /* CTAs of the tensor-core kernel (0 when num_tc_items is 0) */
    int32_t num_warps;         /* warps of the warp kernel (at most one per warp item) */
    int32_t num_slots;         /* split-K partial results, each for one (stream, KV head) */
    int32_t max_page_blocks;   /* page block-table width the plan needs */
    int32_t max_stream_blocks; /* stream block-table width the plan needs */
    int32_t max_stream_slots;  /* most split-K partials of one (stream, KV head) */
    int64_t plan_ints;         /* int32 words in the plan blob */
    int64_t off_stream_page;   /* offsets (int32 words) of the blob's arrays */
    int64_t off_shared_len;
    int64_t off_private_len;
    int64_t off_slot_ptr;
    int64_t off_items;
    int64_t off_page_len;
    int64_t off_cta_ptr;
    int64_t off_warp_ptr;
    int64_t kv_tokens;         /* algorithmic KV tokens read: each page's stream once + all private */
    int64_t off_merge_keys;    /* the (stream, KV head) keys the split-K merge joins; the others have */
    int32_t num_merge_keys;    /* one partial, written as the output directly */
    int32_t reserved;
} padoc_decode_plan;

/* Size in int32 words of the plan blob for these pages and config. */
padoc_status padoc_decode_plan_size(const padoc_page *pages, int32_t num_pages, const padoc_decode_config *cfg,
                                    int64_t *plan_ints);

/* Builds the decode plan (C1's per-branch plan {page, shared_len = P + f_k, private_len} plus the
 * split-K work list and partial-result slots). pages: branch_len = private KV lengths.
 * plan: (host) int32 [capacity_ints]; info: (host) summary.
 * Errors: INVALID_ARGUMENT; UNSUPPORTED for head layouts the kernels do not implement;
 * CAPACITY when capacity_ints is too small. */
padoc_status padoc_build_decode_plan(const padoc_page *pages, int32_t num_pages, const padoc_decode_config *cfg,
                                     int32_t *plan, int64_t capacity_ints, padoc_decode_plan *info);

/* One stream of an explicit stream list (the per-branch plan {page, shared_len = P + f_k,
 * private_len} of C1, given directly instead of derived from padoc_page records). */
typedef struct {
    int32_t page;         /* index into the list's pages; streams are grouped page by page, pages ascending */
    int32_t shared_len;   /* cutoff on the page's shared stream: P + f_k for a branch, the page's whole
                             shared length for its layout stream; 0 <= shared_len <= page_len[page] */
    int32_t private_len;  /* private rows, the newest being the token decoded; 0 for a layout stream */
} padoc_stream_desc;

/* padoc_decode_plan_size / padoc_build_decode_plan for an explicit stream list, as the decoding loop
 * of Algorithm 1 has it at each step: a page's layout stream may have retired while its branches
 * live on, and branches join and leave the batch one by one (App. E.1: a completed stream's row is
 * removed). page_len: (host) int32 [num_pages], the shared-stream tokens of each page in the cache;
 * streams: (host) [num_streams]; cfg->layout_streams must be 0 (the list names every stream). The
 * plan is the one padoc_build_decode_plan gives for the same streams in the same order; Q, out and
 * lse rows follow the list. A page with no stream is skipped.
 * Errors: INVALID_ARGUMENT (also for streams out of page order or a cutoff past page_len);
 * UNSUPPORTED; CAPACITY. */
padoc_status padoc_decode_plan_size_streams(const int32_t *page_len, int32_t num_pages, const padoc_stream_desc *streams,
                                            int32_t num_streams, const padoc_decode_config *cfg, int64_t *plan_ints);
padoc_status padoc_build_decode_plan_streams(const int32_t *page_len, int32_t num_pages,
                                             const padoc_stream_desc *streams, int32_t num_streams,
                                             const padoc_decode_config *cfg, int32_t *plan, int64_t capacity_ints,
                                             padoc_decode_plan *info);

/* Workspace (device) bytes padoc_branch_decode_attn needs for this plan (split-K partials). */
padoc_status padoc_decode_workspace_size(const padoc_decode_plan *info, size_t *bytes);

/* One decode step for every live stream of every page (Alg. 1 "Decode o for all streams using the
 * additive bias A_M", App. E.1): stream s of page p attends to the page's shared stream rows
 * [0, shared_len_s) and to its private rows [0, private_len_s), where the newest private row is
 * the token being decoded.
 *   pool:          the paged KV pool (device pointers inside).
 *   info, plan_dev: host summary and device copy of the plan blob.
 *   page_block_table   (device) int32 [num_pages][page_table_stride], block ids of each page's
 *                      shared stream; stride >= info->max_page_blocks.
 *   stream_block_table (device) int32 [num_streams][stream_table_stride], block ids of each
 *                      stream's private rows; stride >= max(info->max_stream_blocks, 1).
 *   q:   (device) [num_streams][Hq][head_dim] in pool dtype.
 *   out: (device) [num_streams][Hq][head_dim] in pool dtype.  lse: (device) fp32 [num_streams][Hq].
 *   workspace: (device) >= padoc_decode_workspace_size bytes, 256-byte aligned.
 * bf16 path: head_dim 128, Hq / Hkv = 8, block_size 16. f32 path (bring-up): head_dim 64 or 128,
 * any Hq multiple of Hkv, block_size 16; it needs no workspace.
 * Errors: INVALID_ARGUMENT, UNSUPPORTED, WORKSPACE_TOO_SMALL, CUDA. */
padoc_status padoc_branch_decode_attn(const padoc_kv_pool *pool, const padoc_decode_plan *info,
                                      const int32_t *plan_dev, const int32_t *page_block_table,
                                      int32_t page_table_stride, const int32_t *stream_block_table,
                                      int32_t stream_table_stride, const void *q, float scale, void *out,
                                      float *lse, void *workspace, size_t workspace_bytes,
                                      padoc_stream_t stream);

/* Patches a plan built by the planners above, and its host summary, for new private lengths of
 * the same streams (a decoding loop's steady state: every stream appends one token per step and
 * nothing forks or retires): private_len (host) int32 [num_streams] with num_streams =
 * info->num_streams. Each stream keeps its work items and partial slots; the private item that
 * ended at its old length (one per KV head) now ends at the new one, so the plan covers every
 * visible row exactly once as before. O(streams + items). plan is the host copy of the blob (copy
 * it to the device again). Returns CAPACITY, changing nothing, when the patch does not apply (a
 * length below the old one, a stream that had no private rows, an item that would exceed the warp
 * kernel's item length, a chunked-prefill plan): then build a new plan. The stream block table must
 * cover the new lengths (info->max_stream_blocks is updated). Errors: INVALID_ARGUMENT, CAPACITY. */
padoc_status padoc_advance_decode_plan(int32_t *plan, padoc_decode_plan *info, const int32_t *private_len,
                                       int32_t num_streams);

/* One decode step for a caller whose step inputs live in host memory, with no host
 * synchronization: copies stage[0, stage_words) ((host) int32, pinned for an asynchronous copy: the
 * plan blob at word 0, the page block table at off_page_table and the stream block table at
 * off_stream_table, each offset a multiple of 32 words past the blob) to dev_ints ((device) int32
 * [dev_capacity_words], 256-byte aligned) and q_host ((host) [num_streams][Hq][head_dim] in the pool
 * dtype) to q_dev (device, same size), runs padoc_branch_decode_attn on them on `stream`, then
 * copies out_dev and lse_dev into out_host and lse_host ((host), same sizes).
 *   copy_in NULL: everything runs on `stream` (copy_out and the events are not used).
 *   copy_in, copy_out non-NULL (streams) with three events (created by the caller, e.g. with
 *   cudaEventDisableTiming) of the buffer set this call uses: copy_in waits for ev_free (the set's
 *   previous step has copied its results out; record it once before the first use), copies the
 *   inputs in and records ev_in; `stream` waits for ev_in and decodes, and records ev_dec; copy_out
 *   waits for ev_dec, copies the results out and records ev_free. With two buffer sets used in
 *   turn, one step's copies in overlap the previous step's decode and its copies out the next one's.
 * The host buffers must stay unchanged (inputs) or unread (results) until their copies have run.
 * Errors: INVALID_ARGUMENT, and those of padoc_branch_decode_attn. */
padoc_status padoc_launch_decode_step(const padoc_kv_pool *pool, const padoc_decode_plan *info, const int32_t *stage,
                                      int64_t stage_words, int64_t off_page_table, int32_t page_table_stride,
                                      int64_t off_stream_table, int32_t stream_table_stride, int32_t *dev_ints,
                                      int64_t dev_capacity_words, const void *q_host, void *q_dev, float scale,
                                      void *out_dev, float *lse_dev, void *out_host, float *lse_host, void *workspace,
                                      size_t workspace_bytes, padoc_stream_t stream, padoc_stream_t copy_in,
                                      padoc_stream_t copy_out, padoc_event_t ev_free, padoc_event_t ev_in,
                                      padoc_event_t ev_dec);

/* Size of the device array that padoc_branch_decode_attn_noalloc uses as its workspace. */
#define PADOC_STATIC_WORKSPACE_BYTES (32u << 20)

/* padoc_branch_decode_attn for callers that cannot allocate device memory (a plugin inside a
 * framework that owns all device memory and offers it no allocator, or a latency-critical decode
 * loop that must not call cudaMalloc, which may synchronize the device). The paper has no
 * counterpart: it is a deployment convenience of this library.
 * Arguments, layouts and results are those of padoc_branch_decode_attn without the workspace
 * arguments. The split-K partials go to a fixed 256-byte-aligned device array of
 * PADOC_STATIC_WORKSPACE_BYTES (32 MiB) that every GPU which loads this library holds until the
 * process exits; the call allocates nothing (no cudaMalloc, cudaFree or allocating library call).
 *   - The first call on a device looks up that device's address of the array (once per device,
 *     with that device current); make that first call before any stream capture. The address is
 *     kept for the life of the process, so the library must not be used on a device after a
 *     cudaDeviceReset of it (the same holds for the device error word of every call).
 *   - Every call shares the one array, and it keeps the last call's contents. The decode writes
 *     every partial it later reads, so nothing needs clearing, but calls that overlap on the GPU
 *     (other streams, other host threads, concurrent graph launches) race on it: serialize them.
 *   - A plan whose padoc_decode_workspace_size exceeds PADOC_STATIC_WORKSPACE_BYTES is rejected
 *     with PADOC_ERR_WORKSPACE_TOO_SMALL before any launch.
 * Errors: as padoc_branch_decode_attn. */
padoc_status padoc_branch_decode_attn_noalloc(const padoc_kv_pool *pool, const padoc_decode_plan *info,
                                              const int32_t *plan_dev, const int32_t *page_block_table,
                                              int32_t page_table_stride, const int32_t *stream_block_table,
                                              int32_t stream_table_stride, const void *q, float scale, void *out,
                                              float *lse, padoc_stream_t stream);

/* C4: merge of split-K partial softmax results (softmax over a union of disjoint key sets):
 *   lse_r = ln sum_s exp(part_lse[s][r]),  out_r = sum_s exp(part_lse[s][r] - lse_r) part_o[s][r].
 * A part with lse = -inf weighs 0; a row whose parts are all -inf gets lse = -inf and out = 0.
 * part_o: (device) fp32 [num_splits][rows][head_dim]; part_lse: (device) fp32 [num_splits][rows];
 * out: (device) [rows][head_dim] in out_dtype; lse: (device) fp32 [rows] (may be NULL).
 * head_dim a multiple of 4, <= 256. Errors: INVALID_ARGUMENT, CUDA. */
padoc_status padoc_splitk_combine(const float *part_o, const float *part_lse, int32_t num_splits, int64_t rows,
                                  int32_t head_dim, padoc_dtype out_dtype, void *out, float *lse,
                                  padoc_stream_t stream);

/* ============================================================================================
 * FP8 (E4M3) variant of the paged KV cache (C5) and of the decode step (C2)
 * ========================================================================================== */

/* The paper serves a bf16 cache (Sec. 4 serving setup); this variant halves the bytes a decode
 * step reads. K and V are stored as E4M3 codes (the OCP 8-bit format: 4 exponent bits with bias 7,
 * 3 mantissa bits, largest finite 448) with one fp32 scale per (block, KV head); an element's value
 * is code_value * scale. The scale is amax / 448 over the rows the block holds (0 while it holds no
 * nonzero value), so a block's largest magnitude maps to 448. Layouts as padoc_kv_pool:
 *   k_codes, v_codes:   (device) uint8 [num_blocks][num_kv_heads][block_size][head_dim], 16-byte aligned
 *   k_scales, v_scales: (device) fp32 [num_blocks][num_kv_heads]
 * Supported: block_size 16, head_dim 128. */
typedef struct {
    const void *k_codes;
    const void *v_codes;
    const float *k_scales;
    const float *v_scales;
    int32_t num_blocks;
    int32_t block_size;
    int32_t num_kv_heads;
    int32_t head_dim;
} padoc_kv_pool_e4m3;

/* Quantizes whole blocks (a page's prefix after its prefill): (block i, head g) of k_src / v_src
 * ((device) bf16 [count][num_kv_heads][block_size][head_dim]) becomes (block dst_blocks[i], head g)
 * of the pool: scale = amax / 448 (fp32), code = the E4M3 code of x / scale (fp32 division,
 * nearest even, saturating at 448); an all-zero one gets scale 0 and codes 0. dst_blocks: (device)
 * int32 [count]; an id out of range sets the device error word (code 1) and that block is skipped.
 * Errors: INVALID_ARGUMENT, UNSUPPORTED, CUDA. */
padoc_status padoc_quantize_kv_blocks(const padoc_kv_pool_e4m3 *pool, const void *k_src, const void *v_src,
                                      const int32_t *dst_blocks, int32_t count, padoc_stream_t stream);

/* padoc_append_inputs for an E4M3 pool (Algorithm 1's append; sources bf16 [src_total][Hkv][d],
 * queries bf16 as there). Input i goes to row r = slots[i] % block_size of block
 * slots[i] / block_size, every KV head, by the scale rule: the block's scale becomes
 * max(old scale, amax(row) / 448), the old scale taken as 0 when r = 0 (a block's first row starts
 * it afresh; a block handed out again keeps a former owner's scale and rows, which no one reads);
 * when the scale grows from a nonzero old scale, rows 0 .. r-1 are re-encoded (code value x old
 * scale, divided by the new scale, each step rounded to fp32, then encoded nearest even); the row's
 * codes are those of x / new scale. Rows past r are left as they are. The inputs of one call must
 * lie in distinct blocks (Algorithm 1 appends one input per stream, each stream to its own
 * blocks); two inputs in one block race. Errors: INVALID_ARGUMENT, UNSUPPORTED, CUDA. */
padoc_status padoc_append_inputs_e4m3(const padoc_kv_pool_e4m3 *pool, const void *k_src, const void *v_src,
                                      const void *q_src, int64_t src_total, int32_t num_q_heads, void *q_dst,
                                      const int32_t *src_rows, const int32_t *slots, int32_t count,
                                      padoc_stream_t stream);

/* padoc_branch_decode_attn over an E4M3 pool: the same plans (padoc_build_decode_plan and the other
 * planners, built with the same padoc_decode_config), tables, workspace and results; q, out bf16
 * [num_streams][Hq][128], lse fp32. Attention is over the dequantized values code_value * scale:
 * codes become bf16 exactly in shared memory, the K scale multiplies each 16-token block's scores
 * and the V scale the block's probabilities in fp32 before they are rounded to bf16. Hq / Hkv = 8,
 * block_size 16, head_dim 128. Errors: INVALID_ARGUMENT, UNSUPPORTED, WORKSPACE_TOO_SMALL, CUDA. */
padoc_status padoc_branch_decode_attn_e4m3(const padoc_kv_pool_e4m3 *pool, const padoc_decode_plan *info,
                                           const int32_t *plan_dev, const int32_t *page_block_table,
                                           int32_t page_table_stride, const int32_t *stream_block_table,
                                           int32_t stream_table_stride, const void *q, float scale, void *out,
                                           float *lse, void *workspace, size_t workspace_bytes,
                                           padoc_stream_t stream);

/* ============================================================================================
 * Branch prefill over the paged cache: chunks of several query tokens per stream
 * ========================================================================================== */

/* A chunk of consecutive query tokens of one stream whose K/V rows are already in the paged cache
 * (App. E.2: a child's branch-initialization input and its residual prefill; Sec. 3.2 visibility).
 * Chunks are processed by the decode kernels with the chunk's tokens as streams of its page: each
 * page's shared stream is read once per group of up to 32 tokens of a chunk, and a chunk's own
 * private rows once per group on the tensor cores (8 or more tokens) instead of once per token. */
typedef struct {
    int32_t page;           /* index into the call's pages; chunks grouped page by page, pages ascending */
    int32_t shared_len;     /* branch chunk: the stream's cutoff on the page's shared stream (P + f_k);
                               shared-stream chunk: the shared rows before the chunk's first token */
    int32_t private_start;  /* branch chunk: the stream's private rows before the chunk (its first token
                               is private row private_start); -1: the chunk's tokens are the shared-stream
                               rows shared_len .. shared_len + num_tokens - 1 (prefix or layout tokens) */
    int32_t num_tokens;     /* >= 1 */
} padoc_prefill_chunk;

/* Plan for a chunked prefill, run by padoc_branch_decode_attn (the same kernels, Q / out / lse rows =
 * the chunks' tokens in order). Token i of a branch chunk attends to shared rows [0, shared_len) and
 * private rows [0, private_start + i + 1) (causal inside the chunk); token i of a shared-stream chunk
 * to shared rows [0, shared_len + i + 1). page_len: (host) int32 [num_pages], each page's shared rows
 * in the cache; chunks: (host) [num_chunks]. The stream block table passed to the decode call has
 * one row per token, every token of a branch chunk carrying its stream's private blocks
 * (padoc_expand_chunk_table writes it from one row per chunk). cfg->layout_streams must be 0.
 * Errors: INVALID_ARGUMENT (also chunks out of page order, a cutoff past page_len, a shared-stream
 * chunk reaching past page_len); UNSUPPORTED; CAPACITY. */
padoc_status padoc_chunk_prefill_plan_size(const int32_t *page_len, int32_t num_pages, const padoc_prefill_chunk *chunks,
                                           int32_t num_chunks, const padoc_decode_config *cfg, int64_t *plan_ints);
padoc_status padoc_build_chunk_prefill_plan(const int32_t *page_len, int32_t num_pages,
                                            const padoc_prefill_chunk *chunks, int32_t num_chunks,
                                            const padoc_decode_config *cfg, int32_t *plan, int64_t capacity_ints,
                                            padoc_decode_plan *info);

/* Writes the per-token stream block table of a chunked prefill: chunk_table (host) int32
 * [num_chunks][chunk_stride] holds each chunk's private block ids (any content for a shared-stream
 * chunk); row r of stream_table (host) int32 [capacity_rows][stream_stride] gets the row of the
 * chunk that token r belongs to, padded with -1. Errors: INVALID_ARGUMENT; CAPACITY when
 * capacity_rows is below the chunks' token count. */
padoc_status padoc_expand_chunk_table(const padoc_prefill_chunk *chunks, int32_t num_chunks, const int32_t *chunk_table,
                                      int32_t chunk_stride, int32_t *stream_table, int32_t stream_stride,
                                      int64_t capacity_rows);

/* ============================================================================================
 * Algorithm 1 (App. E.1): the masked parallel decoding loop over the paged cache
 * ========================================================================================== */

/* Host-side scheduler state of the loop for a batch of pages sharing one KV pool (opaque; created by
 * padoc_mpd_create, freed by padoc_mpd_destroy, in host memory). It keeps, per page, the shared stream's blocks (prefix X, then the layout stream's
 * tokens) and, per stream, its cutoff on the shared stream and its private blocks, and it hands out
 * and takes back pool blocks. It realises the logical mask M of App. E.1 without materialising it:
 *   - each step appends one input per live stream (M <- [M I_C]): the layout stream's input extends
 *     the page's shared stream, a branch's input extends its private rows;
 *   - a fork copies the layout stream's pre-boundary row: the new branch's cutoff is the page's
 *     shared length at that moment (P + the layout tokens in the cache), and it appends its
 *     branch-initialization input at the next step;
 *   - a retired branch's private blocks return to the pool; a page's shared blocks return when its
 *     last stream retires (a completed stream's row is removed and its positions are never read
 *     again).
 * Streams of a step are ordered page by page (pages in admission order), within a page its live
 * branches in fork order, then its layout stream while it is live. Stream ids count up from 0 in
 * creation order over the object's life. Not thread-safe: one caller at a time. */
typedef struct padoc_mpd padoc_mpd;

/* num_blocks pool blocks of block_size (16) tokens, handed out first in the order of block_order
 * ((host) int32 [num_blocks], a permutation of 0..num_blocks-1; NULL = ascending); returned blocks
 * are handed out again after those (first in, first out). Errors: INVALID_ARGUMENT, UNSUPPORTED. */
padoc_status padoc_mpd_create(int32_t num_blocks, int32_t block_size, const int32_t *block_order, padoc_mpd **mpd);
void padoc_mpd_destroy(padoc_mpd *mpd);

/* Admits a page whose prefix X has prefix_len tokens (Algorithm 1: "Prefill X; initialize the
 * layout stream"). prefix_slots: (host) int32 [prefix_len] receives the pool slot
 * (block * block_size + offset) of each prefix token; the caller writes the prefix K/V there
 * (padoc_append_inputs) before the first step that decodes the page. The prefill's output decides
 * the first events: num_forks branches forked from the prefill (f = 0: they see X only) and
 * layout_eos = 1 when the layout stream ends at once. new_streams: (host) int32 [1 + num_forks]
 * receives the layout stream's id (-1 with layout_eos) and then the new branches' ids.
 * page_id: (host) the page's id (admission counter). Errors: INVALID_ARGUMENT (also during a step,
 * between padoc_mpd_begin_step and padoc_mpd_end_step); CAPACITY when the pool has too few free
 * blocks (nothing changes). */
padoc_status padoc_mpd_add_page(padoc_mpd *mpd, int32_t prefix_len, int32_t num_forks, int32_t layout_eos,
                                int32_t *page_id, int32_t *prefix_slots, int32_t *new_streams);

/* Begins one step: "Let C be the live-stream count and i their next inputs. Append i to the cache"
 * (Algorithm 1). Every live stream gets the pool slot of its next input (a new block when its next
 * row starts one); its length counts that input from now on. stream_ids, append_slots: (host) int32
 * [capacity] receive the step's streams in order and their slots; num_streams: C.
 * Errors: INVALID_ARGUMENT (null pointers, a step already begun); CAPACITY when capacity < C or the
 * pool has too few free blocks (nothing changes). */
padoc_status padoc_mpd_begin_step(padoc_mpd *mpd, int32_t *num_streams, int32_t *stream_ids, int32_t *append_slots,
                                  int32_t capacity);

/* Sizes of the current step's decode tables: live pages, live streams, the widest page and stream
 * block lists. Valid between padoc_mpd_begin_step and padoc_mpd_end_step. */
padoc_status padoc_mpd_step_shape(const padoc_mpd *mpd, int32_t *num_pages, int32_t *num_streams,
                                  int32_t *max_page_blocks, int32_t *max_stream_blocks);

/* The current step's decode inputs, in step order: page_len (host) int32 [num_pages] and streams
 * (host) [num_streams] for padoc_build_decode_plan_streams, and the block tables for
 * padoc_branch_decode_attn: page_table (host) int32 [num_pages][page_stride], stream_table (host)
 * int32 [num_streams][stream_stride], unused entries -1. Strides at least the step_shape widths
 * (stream_stride >= 1). Errors: INVALID_ARGUMENT (also outside a step). */
padoc_status padoc_mpd_step_tables(const padoc_mpd *mpd, int32_t *page_len, padoc_stream_desc *streams,
                                   int32_t *page_table, int32_t page_stride, int32_t *stream_table,
                                   int32_t stream_stride);

/* Ends the step with each stream's output event, in step order ((host) arrays [num_streams], the
 * C of padoc_mpd_begin_step): num_forks[i] branches forked from stream i's output ("the layout
 * output completes region B_k": only a layout stream forks; NULL = none), eos[i] != 0 when stream
 * i's output is EOS (it retires; NULL = none). A layout stream may fork and retire on the same
 * output. new_streams: (host) int32 [capacity] receives the new branches' ids (in step order, a
 * stream's forks consecutively), num_new their count. Errors: INVALID_ARGUMENT (no step begun, a
 * wrong count, a branch that forks); CAPACITY when capacity is below the new branches (nothing
 * changes). */
padoc_status padoc_mpd_end_step(padoc_mpd *mpd, const int32_t *num_forks, const uint8_t *eos, int32_t num_streams,
                                int32_t *new_streams, int32_t capacity, int32_t *num_new);

/* Layout of one step prepared by padoc_mpd_prepare_step in the caller's int32 staging buffer
 * (offsets in int32 words, each a multiple of 32, so every part starts on a 128-byte boundary). */
typedef struct {
    int32_t num_streams;       /* C: the step's streams */
    int32_t num_pages;         /* live pages (rows of the page table) */
    int32_t page_stride;       /* page-table row width (>= 1) */
    int32_t stream_stride;     /* stream-table row width (>= 1) */
    int64_t off_plan;          /* the decode plan blob (plan.plan_ints words) */
    int64_t off_page_table;    /* int32 [num_pages][page_stride], unused entries -1 */
    int64_t off_stream_table;  /* int32 [num_streams][stream_stride], unused entries -1 */
    int64_t off_slots;         /* int32 [num_streams]: each stream's append slot */
    int64_t off_rows;          /* int32 [num_streams]: left for the caller (e.g. the source rows of the
                                  inputs for padoc_append_inputs), not written */
    int64_t off_first_blocks;  /* int32 [plan.num_warps][4]: the pool rows ((block id x Hkv + KV head) x
                                  block_size) of the first four 16-token blocks of each warp list's
                                  first item, -2 - row for the block holding its stream's newest row,
                                  -1 past its end; padoc_mpd_launch_step's decode warps start these
                                  blocks before they read their item headers */
    int64_t off_stream_ids;    /* int32 [num_streams]: the step's stream ids (host use) */
    int64_t upload_words;      /* [0, upload_words) is what the device needs: everything but the ids */
    int64_t total_words;       /* words the step needs in the staging buffer */
    padoc_decode_plan plan;    /* host summary of the step's decode plan */
} padoc_mpd_step;

/* One call for a step's host work: padoc_mpd_begin_step, padoc_mpd_step_tables and
 * padoc_build_decode_plan_streams (with cfg; cfg->layout_streams 0) in one planner pass, written
 * into stage ((host) int32 [capacity_words], e.g. pinned memory for one host->device copy) in the
 * layout `step` describes. With too small a capacity it returns CAPACITY with step->total_words
 * set and begins nothing; so does a pool without enough free blocks (step->total_words = 0).
 * Errors: INVALID_ARGUMENT (also a step already begun), UNSUPPORTED, CAPACITY. */
padoc_status padoc_mpd_prepare_step(padoc_mpd *mpd, const padoc_decode_config *cfg, int32_t *stage,
                                    int64_t capacity_words, padoc_mpd_step *step);

/* Runs a step prepared by padoc_mpd_prepare_step, all on `stream`, with no host synchronization:
 * copies stage[0, step->upload_words) (host; pinned memory makes the copy asynchronous, and the
 * stage must stay unchanged until the copy has run; NULL: dev_ints already holds those words) to
 * dev_ints ((device) int32 [dev_capacity_words], 256-byte aligned), appends every input (padoc_append_inputs with the step's
 * slots and the source rows the caller wrote at stage[step->off_rows]; k_src / v_src
 * [src_total][Hkv][d], q_src [src_total][Hq][d], q_dst (device) [C][Hq][d] receives the step's
 * queries) and decodes every stream (padoc_branch_decode_attn: out [C][Hq][d], lse fp32 [C][Hq],
 * workspace >= padoc_decode_workspace_size(&step->plan) bytes). The decode is launched behind the
 * append with programmatic dependent launch, and its warps without tensor-core work read the plan,
 * the block tables and the paged blocks that hold no stream's newest row before they wait for the
 * append. Nothing is launched for C = 0.
 * Errors: INVALID_ARGUMENT (also dev_capacity_words < upload_words), UNSUPPORTED,
 * WORKSPACE_TOO_SMALL, CUDA. */
padoc_status padoc_mpd_launch_step(const padoc_mpd_step *step, const int32_t *stage, int32_t *dev_ints,
                                   int64_t dev_capacity_words, const padoc_kv_pool *pool, const void *k_src,
                                   const void *v_src, const void *q_src, int64_t src_total, void *q_dst, float scale,
                                   void *out, float *lse, void *workspace, size_t workspace_bytes,
                                   padoc_stream_t stream);

/* The loop's per-step host work behind one call (Algorithm 1, App. E.1: "decode all live streams"
 * once per iteration): a runner keeps, for one scheduler and one pool, two pinned staging buffers
 * used in turn (a step's buffer is reused two steps later, after the event recorded behind that
 * step's launches has completed), the device copy of the step's ints, the step's query buffer and
 * the decode workspace. It allocates them (cudaHostAlloc / cudaMalloc) as the steps need and frees
 * them in padoc_mpd_runner_destroy; to replace a device buffer it first waits for the step's
 * stream. The scheduler and the pool must outlive the runner; cfg->layout_streams must be 0.
 * Errors: INVALID_ARGUMENT (mismatched block size, KV heads or head_dim, a pool with fewer blocks
 * than the scheduler), CUDA. */
typedef struct padoc_mpd_runner padoc_mpd_runner;
padoc_status padoc_mpd_runner_create(padoc_mpd *mpd, const padoc_decode_config *cfg, const padoc_kv_pool *pool,
                                     padoc_mpd_runner **runner);
void padoc_mpd_runner_destroy(padoc_mpd_runner *runner);

/* Arguments of padoc_mpd_runner_step, kept by the caller from step to step. */
typedef struct {
    const void *k_src;                  /* (device) [src_total][Hkv][d]: the inputs' K rows, pool dtype */
    const void *v_src;                  /* (device) [src_total][Hkv][d] */
    const void *q_src;                  /* (device) [src_total][Hq][d] */
    int64_t src_total;
    const int32_t *src_row_of_stream;   /* (host) int32 [num_stream_ids]: the source row of each live
                                           stream's next input, indexed by stream id */
    int32_t num_stream_ids;             /* at least the number of stream ids created so far */
    float scale;                        /* softmax scale */
    void *out;                          /* (device) [out_rows][Hq][d], pool dtype: rows [0, C) receive the
                                           step's outputs in step order */
    float *lse;                         /* (device) fp32 [out_rows][Hq] */
    int32_t out_rows;
    int32_t ids_capacity;
    int32_t *stream_ids;                /* (host) int32 [ids_capacity]: receives the step's stream ids */
    padoc_stream_t stream;              /* every copy and launch of the step goes here */
} padoc_mpd_run_args;

/* One step: padoc_mpd_prepare_step into the runner's next staging buffer, the source row of each
 * stream's input from a->src_row_of_stream, then padoc_mpd_launch_step with the runner's buffers,
 * and an event behind it; no host synchronization except the wait for the staging buffer's copy of
 * two steps ago (and, when a buffer grows, for the stream). num_streams: C (0: nothing launched);
 * upload_bytes (NULL allowed): the bytes copied to the device for the step.
 * The step stays begun until padoc_mpd_end_step. Errors: CAPACITY when out_rows or ids_capacity is
 * below the live streams, or the pool lacks free blocks (nothing begins); INVALID_ARGUMENT (also a
 * step already begun, num_stream_ids too small; nothing begins); past the planning (CUDA,
 * UNSUPPORTED) the step has begun and the caller ends it. Source rows out of range set the device
 * error word (padoc_append_inputs). */
padoc_status padoc_mpd_runner_step(padoc_mpd_runner *runner, const padoc_mpd_run_args *args, int32_t *num_streams,
                                   int64_t *upload_bytes);

/* The last step the runner prepared and its staging buffer (valid until the runner's step after
 * next): for callers that keep a record of the steps. Errors: INVALID_ARGUMENT (no step yet). */
padoc_status padoc_mpd_runner_last_step(const padoc_mpd_runner *runner, padoc_mpd_step *step, const int32_t **stage);

/* Live pages, live streams and free pool blocks. */
padoc_status padoc_mpd_status(const padoc_mpd *mpd, int32_t *live_pages, int32_t *live_streams, int32_t *free_blocks);

/* Writes one step's inputs (device): for i < count, the K and V rows src_rows[i] of k_src / v_src
 * ([src_total][Hkv][head_dim]) go to pool slot slots[i] (block slots[i] / block_size, row
 * slots[i] % block_size, every KV head), and, when q_src is not NULL, Q row src_rows[i] of q_src
 * ([src_total][num_q_heads][head_dim]) goes to row i of q_dst ([count][num_q_heads][head_dim]), the
 * decode call's query order. src_rows NULL means row i. The pool's K and V arrays are written;
 * everything is in the pool's dtype, 16-byte aligned. Used for the prefix of a new page and for
 * every step's inputs (Algorithm 1's append). A slot or source row out of range sets the device
 * error word (code 1) and that row is skipped. Errors: INVALID_ARGUMENT, UNSUPPORTED, CUDA. */
padoc_status padoc_append_inputs(const padoc_kv_pool *pool, const void *k_src, const void *v_src, const void *q_src,
                                 int64_t src_total, int32_t num_q_heads, void *q_dst, const int32_t *src_rows,
                                 const int32_t *slots, int32_t count, padoc_stream_t stream);

/* ============================================================================================
 * C3: packed variable-length ancestor prefill (training forward / branch prefill)
 * ========================================================================================== */

/* Every packed token is a query under the ancestor rule (App. C.1: the causal problem over M and
 * one bottom-right-aligned causal problem per branch over [K_{M<=f_k}; K_{Y_k}], computed in
 * packed order without any gather). Fully masked tiles are skipped via the tile map.
 *   q: (device) [T][Hq][head_dim]; k, v: (device) [T][Hkv][head_dim]; all in dtype, 16-byte aligned.
 *   spans_dev: (device) int32 [T][4] from padoc_build_query_spans.
 *   tile_row_ptr_dev / tile_k_dev / tile_kind_dev: (device) the tile map from
 *   padoc_build_tile_map built with (q_tile, k_tile) = padoc_prefill_tile_shape(dtype, head_dim)
 *   (the f32 path reads only the spans and accepts NULL tile pointers).
 *   out: (device) [T][Hq][head_dim] in dtype; lse: (device) fp32 [T][Hq].
 * bf16 path: head_dim 128, Hq a multiple of Hkv. f32 path: head_dim 64 or 128.
 * Errors: INVALID_ARGUMENT, UNSUPPORTED, CUDA. */
padoc_status padoc_ancestor_prefill_attn(const void *q, const void *k, const void *v, padoc_dtype dtype,
                                         int64_t total_tokens, int32_t num_q_heads, int32_t num_kv_heads,
                                         int32_t head_dim, const int32_t *spans_dev,
                                         const int32_t *tile_row_ptr_dev, const int32_t *tile_k_dev,
                                         const int8_t *tile_kind_dev, int32_t q_tile, int32_t k_tile,
                                         float scale, void *out, float *lse, padoc_stream_t stream);

/* ============================================================================================
 * Prefill backward: gradients of C3 (training backward of the tree-varlen attention)
 * ========================================================================================== */

/* A tile map in device memory (host struct of device pointers). Query-major maps come from
 * padoc_build_tile_map (ptr = row_ptr, idx = k_tiles, order = NULL); key-major maps from
 * padoc_build_key_tile_map (ptr = col_ptr, idx = q_tiles, order = k_order). */
typedef struct {
    const int32_t *ptr;
    const int32_t *idx;
    const int8_t *kind;
    const int32_t *order;
    int32_t q_tile, k_tile;
} padoc_tile_map_dev;

/* Workspace of padoc_ancestor_prefill_bwd: two fp32 arrays [Hq][ceil(T/128)*128] (per head the
 * negated base-2 log-sum-exp of the forward and D = rowsum(dO * O)), then 2048 bytes per padded row
 * for the fp32 partials of the heaviest key tiles, whose gradients two CTAs share; 256-byte aligned. */
padoc_status padoc_prefill_bwd_workspace_size(int64_t total_tokens, int32_t num_q_heads, size_t *bytes);

/* Gradients of the packed ancestor prefill for an upstream gradient dO (App. C.1; Sec. 3.2
 * visibility). Per query row and head, with P_j = exp(scale * q.k_j - lse) over the visible keys:
 *   D = sum_c dO[c] O[c],  dS_j = P_j (dO.v_j - D),  dQ = scale * sum_j dS_j k_j;
 * every key of KV head g collects over the queries that see it and the query heads reading g:
 *   dK_j = scale * sum dS_ij q_i,  dV_j = sum P_ij dO_i,
 * so a shared-stream key's gradient sums over the stream's later tokens and over every branch
 * forked after it (the scatter-add of the gather's backward), with no gather and no atomics.
 *   q, out, dout: (device) [T][Hq][head_dim]; k, v: (device) [T][Hkv][head_dim]; all in dtype,
 *   16-byte aligned; out and lse are the forward's outputs (lse natural log, fp32 [T][Hq]).
 *   spans_dev: (device) int32 [T][4] from padoc_build_query_spans.
 *   q_map: query-major map, k_map: key-major map, built with padoc_prefill_bwd_tile_shapes.
 *   dq: (device) [T][Hq][head_dim]; dk, dv: (device) [T][Hkv][head_dim]; in dtype. Every row is
 *   written (a key no query sees would get zeros; in the packed layout every token sees itself).
 *   workspace: (device) padoc_prefill_bwd_workspace_size bytes, 256-byte aligned.
 * bf16 path: head_dim 128, tensor cores. f32 path: head_dim 64 or 128 (bring-up, CUDA cores).
 * Errors: INVALID_ARGUMENT, UNSUPPORTED, WORKSPACE_TOO_SMALL, CUDA. */
padoc_status padoc_ancestor_prefill_bwd(const void *q, const void *k, const void *v, const void *out,
                                        const void *dout, const float *lse, padoc_dtype dtype, int64_t total_tokens,
                                        int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                        const int32_t *spans_dev, const padoc_tile_map_dev *q_map,
                                        const padoc_tile_map_dev *k_map, float scale, void *dq, void *dk, void *dv,
                                        void *workspace, size_t workspace_bytes, padoc_stream_t stream);

/* ============================================================================================
 * Status
 * ========================================================================================== */

/* Self-check of the tensor-core encodings the bf16 kernels rely on (no counterpart in the paper:
 * a hardware check a caller may run once per device). With a, bk, v (device) bf16 [128][128]
 * row-major, computes on one CTA with tcgen05 MMAs whose operands sit in 128-byte-swizzled shared
 * memory: c1 = a . bk^T (both operands K-major), c2 = a . v (v as an MN-major operand) and
 * c3 = a . v with a read from tensor memory, fp32 [128][128] row-major (device). The caller
 * compares them with its own product. Errors: INVALID_ARGUMENT, CUDA. */
padoc_status padoc_selftest_tcgen05(const void *a, const void *bk, const void *v, float *c1, float *c2, float *c3,
                                    padoc_stream_t stream);

/* Self-check of the failure path every kernel's waits share (no counterpart in the paper: the
 * library's own failure detection). One CTA of 64 threads waits, with the same bounded mbarrier
 * wait the kernels use but a limit of limit_us microseconds (1 .. 100000), on a barrier that nothing
 * ever arrives at. The wait gives up, records code 2 (bounded wait ran out) with `site` as the
 * detail in the device error word, and every thread that gave up adds 1 to *gave_up ((device)
 * int32, which the caller zeroes first); the kernel then returns, nothing being in flight, and the
 * context stays usable. Read the error with padoc_check_device_errors.
 * Errors: INVALID_ARGUMENT, CUDA. */
padoc_status padoc_selftest_wait_timeout(int32_t limit_us, int32_t site, int32_t *gave_up, padoc_stream_t stream);

/* Synchronizes `stream`, then reads and clears the current device's error word. Returns
 * PADOC_ERR_DEVICE_CHECK if a kernel recorded a failed check since the last call (code and detail
 * via padoc_last_device_error), PADOC_ERR_CUDA if the stream reports an error, else PADOC_OK. */
padoc_status padoc_check_device_errors(padoc_stream_t stream);

/* The code and detail of the device error found by the last padoc_check_device_errors on this
 * thread: code 1 = block id out of range (detail = the id), 2 = bounded wait ran out
 * (detail = the kernel's wait site), 3 = a kernel's dynamic shared memory did not start on the
 * 1024-byte boundary its swizzled tiles need (detail = the start address mod 1024; the kernel did
 * no work). */
void padoc_last_device_error(int32_t *code, int32_t *detail);

const char *padoc_status_string(padoc_status status);
int32_t padoc_version(void);

#ifdef __cplusplus
}
#endif

#endif /* PADOC_ATTN_H */
