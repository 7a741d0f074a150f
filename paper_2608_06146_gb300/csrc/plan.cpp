// plan.cpp -- C1: ancestor descriptors, prefill tile map and decode plan (host, integer only).
//
// The visibility rule is the packed form of the ancestor sets (Sec. 3.2; App. C.1): within a page
// [X | layout | Y_1..Y_N], a prefix or layout token q sees [page_begin, q]; a branch token of Y_k
// sees [page_begin, page_begin + P + f_k) and [ybase_k, q]. Everything here is exact integer
// arithmetic; outputs are bit-exact and canonical (see padoc_attn.h).
#include <algorithm>
#include <atomic>
#include <cstdint>
#include <cstring>
#include <numeric>
#include <queue>
#include <vector>

#include <cuda_runtime.h>

#include "padoc_attn.h"
#include "plan_internal.h"
#include "plan_build.h"

namespace {

padoc_status validate_pages(const padoc_page *pages, int32_t num_pages, int64_t *total)
{
    if (num_pages < 0 || (num_pages > 0 && pages == nullptr)) return PADOC_ERR_INVALID_ARGUMENT;
    int64_t t = 0;
    for (int32_t p = 0; p < num_pages; ++p) {
        const padoc_page &pg = pages[p];
        if (pg.prefix_len < 0 || pg.layout_len < 0 || pg.num_branches < 0) return PADOC_ERR_INVALID_ARGUMENT;
        if (pg.num_branches > 0 && (pg.fork_offset == nullptr || pg.branch_len == nullptr))
            return PADOC_ERR_INVALID_ARGUMENT;
        int64_t s = (int64_t)pg.prefix_len + pg.layout_len;
        for (int32_t k = 0; k < pg.num_branches; ++k) {
            if (pg.fork_offset[k] < 0 || pg.fork_offset[k] > pg.layout_len) return PADOC_ERR_INVALID_ARGUMENT;
            if (pg.branch_len[k] < 1) return PADOC_ERR_INVALID_ARGUMENT;
            s += pg.branch_len[k];
        }
        if (s < 1) return PADOC_ERR_INVALID_ARGUMENT;
        t += s;
        if (t >= (int64_t)INT32_MAX) return PADOC_ERR_INVALID_ARGUMENT;
    }
    if (total) *total = t;
    return PADOC_OK;
}

void fill_spans(const padoc_page *pages, int32_t num_pages, int32_t *spans)
{
    int64_t pb = 0;
    for (int32_t p = 0; p < num_pages; ++p) {
        const padoc_page &pg = pages[p];
        const int64_t M = (int64_t)pg.prefix_len + pg.layout_len;
        for (int64_t q = 0; q < M; ++q) {   // one causal stream over [X | layout]
            int32_t *o = spans + 4 * (pb + q);
            o[0] = (int32_t)pb;
            o[1] = (int32_t)(pb + q + 1);
            o[2] = o[1];
            o[3] = o[1];
        }
        int64_t ybase = pb + M;
        for (int32_t k = 0; k < pg.num_branches; ++k) {
            const int32_t vis_end = (int32_t)(pb + pg.prefix_len + pg.fork_offset[k]);
            for (int32_t i = 0; i < pg.branch_len[k]; ++i) {
                int32_t *o = spans + 4 * (ybase + i);
                o[0] = (int32_t)pb;
                o[1] = vis_end;
                o[2] = (int32_t)ybase;
                o[3] = (int32_t)(ybase + i + 1);
            }
            ybase += pg.branch_len[k];
        }
        pb = ybase;
    }
}

// Walks the tile map; emit(qt, kt, kind) is called in ascending (qt, kt) order.
template <class Emit>
void walk_tiles(const int32_t *spans, int64_t T, int32_t q_tile, int32_t k_tile, Emit emit)
{
    const int64_t nkt = (T + k_tile - 1) / k_tile;
    std::vector<int64_t> cnt((size_t)std::max<int64_t>(nkt, 1), 0);
    std::vector<int32_t> touched;
    const int64_t nqt = (T + q_tile - 1) / q_tile;
    for (int64_t qt = 0; qt < nqt; ++qt) {
        const int64_t r0 = qt * q_tile, r1 = std::min<int64_t>(T, r0 + q_tile);
        touched.clear();
        for (int64_t r = r0; r < r1; ++r) {
            for (int s = 0; s < 2; ++s) {
                const int64_t a = spans[4 * r + 2 * s], b = spans[4 * r + 2 * s + 1];
                if (b <= a) continue;
                for (int64_t kt = a / k_tile; kt <= (b - 1) / k_tile; ++kt) {
                    const int64_t lo = std::max<int64_t>(a, kt * k_tile), hi = std::min<int64_t>(b, (kt + 1) * k_tile);
                    if (cnt[kt] == 0) touched.push_back((int32_t)kt);
                    cnt[kt] += hi - lo;
                }
            }
        }
        std::sort(touched.begin(), touched.end());
        const int64_t full = (r1 - r0) * (int64_t)k_tile;
        for (int32_t kt : touched) {
            emit(qt, kt, cnt[kt] == full ? (int8_t)PADOC_TILE_FULL : (int8_t)PADOC_TILE_PARTIAL);
            cnt[kt] = 0;
        }
    }
}

}  // namespace

extern "C" padoc_status padoc_packed_size(const padoc_page *pages, int32_t num_pages, int64_t *total_tokens)
{
    if (!total_tokens) return PADOC_ERR_INVALID_ARGUMENT;
    return validate_pages(pages, num_pages, total_tokens);
}

extern "C" padoc_status padoc_build_query_spans(const padoc_page *pages, int32_t num_pages, int32_t *spans,
                                                int64_t capacity_tokens)
{
    int64_t T = 0;
    padoc_status st = validate_pages(pages, num_pages, &T);
    if (st != PADOC_OK) return st;
    if (T > 0 && !spans) return PADOC_ERR_INVALID_ARGUMENT;
    if (capacity_tokens < T) return PADOC_ERR_CAPACITY;
    fill_spans(pages, num_pages, spans);
    return PADOC_OK;
}

extern "C" padoc_status padoc_prefill_tile_shape(padoc_dtype dtype, int32_t head_dim, int32_t *q_tile,
                                                 int32_t *k_tile)
{
    if (!q_tile || !k_tile) return PADOC_ERR_INVALID_ARGUMENT;
    if (dtype == PADOC_DTYPE_BF16 && head_dim == 128) { *q_tile = PADOC_PREFILL_Q_TILE; *k_tile = PADOC_PREFILL_K_TILE; return PADOC_OK; }
    if (dtype == PADOC_DTYPE_F32 && (head_dim == 64 || head_dim == 128)) { *q_tile = PADOC_PREFILL_Q_TILE; *k_tile = PADOC_PREFILL_K_TILE; return PADOC_OK; }
    return PADOC_ERR_UNSUPPORTED;
}

extern "C" padoc_status padoc_tile_map_size(const padoc_page *pages, int32_t num_pages, int32_t q_tile,
                                            int32_t k_tile, int64_t *num_q_tiles, int64_t *nnz)
{
    int64_t T = 0;
    padoc_status st = validate_pages(pages, num_pages, &T);
    if (st != PADOC_OK) return st;
    if (q_tile < 1 || k_tile < 1 || !num_q_tiles || !nnz) return PADOC_ERR_INVALID_ARGUMENT;
    std::vector<int32_t> spans((size_t)std::max<int64_t>(T, 1) * 4);
    fill_spans(pages, num_pages, spans.data());
    int64_t n = 0;
    walk_tiles(spans.data(), T, q_tile, k_tile, [&](int64_t, int32_t, int8_t) { ++n; });
    *num_q_tiles = (T + q_tile - 1) / q_tile;
    *nnz = n;
    return PADOC_OK;
}

extern "C" padoc_status padoc_build_tile_map(const padoc_page *pages, int32_t num_pages, int32_t q_tile,
                                             int32_t k_tile, int32_t *row_ptr, int32_t *k_tiles, int8_t *kinds,
                                             int64_t capacity_nnz)
{
    int64_t T = 0;
    padoc_status st = validate_pages(pages, num_pages, &T);
    if (st != PADOC_OK) return st;
    if (q_tile < 1 || k_tile < 1 || !row_ptr) return PADOC_ERR_INVALID_ARGUMENT;
    std::vector<int32_t> spans((size_t)std::max<int64_t>(T, 1) * 4);
    fill_spans(pages, num_pages, spans.data());
    int64_t n = 0;
    walk_tiles(spans.data(), T, q_tile, k_tile, [&](int64_t, int32_t, int8_t) { ++n; });
    if (n > capacity_nnz) return PADOC_ERR_CAPACITY;
    if (n > 0 && (!k_tiles || !kinds)) return PADOC_ERR_INVALID_ARGUMENT;
    const int64_t nqt = (T + q_tile - 1) / q_tile;
    for (int64_t i = 0; i <= nqt; ++i) row_ptr[i] = 0;
    int64_t e = 0;
    walk_tiles(spans.data(), T, q_tile, k_tile, [&](int64_t qt, int32_t kt, int8_t kind) {
        k_tiles[e] = kt;
        kinds[e] = kind;
        ++e;
        row_ptr[qt + 1] = (int32_t)e;
    });
    for (int64_t i = 1; i <= nqt; ++i) row_ptr[i] = std::max(row_ptr[i], row_ptr[i - 1]);
    return PADOC_OK;
}

extern "C" padoc_status padoc_build_key_tile_map(const padoc_page *pages, int32_t num_pages, int32_t q_tile,
                                                 int32_t k_tile, int32_t *col_ptr, int32_t *q_tiles, int8_t *kinds,
                                                 int32_t *k_order, int64_t capacity_nnz)
{
    int64_t T = 0;
    padoc_status st = validate_pages(pages, num_pages, &T);
    if (st != PADOC_OK) return st;
    if (q_tile < 1 || k_tile < 1 || !col_ptr || !k_order) return PADOC_ERR_INVALID_ARGUMENT;
    std::vector<int32_t> spans((size_t)std::max<int64_t>(T, 1) * 4);
    fill_spans(pages, num_pages, spans.data());
    const int64_t nkt = (T + k_tile - 1) / k_tile;
    std::vector<int64_t> cnt((size_t)nkt + 1, 0);
    int64_t n = 0;
    walk_tiles(spans.data(), T, q_tile, k_tile, [&](int64_t, int32_t kt, int8_t) { ++cnt[(size_t)kt + 1]; ++n; });
    if (n > capacity_nnz) return PADOC_ERR_CAPACITY;
    if (n > 0 && (!q_tiles || !kinds)) return PADOC_ERR_INVALID_ARGUMENT;
    for (int64_t c = 0; c < nkt; ++c) cnt[(size_t)c + 1] += cnt[(size_t)c];
    for (int64_t c = 0; c <= nkt; ++c) col_ptr[c] = (int32_t)cnt[(size_t)c];
    // the walk visits q-tiles in ascending order, so each column's entries come out ascending
    std::vector<int64_t> fill(cnt.begin(), cnt.end() - 1);
    walk_tiles(spans.data(), T, q_tile, k_tile, [&](int64_t qt, int32_t kt, int8_t kind) {
        const int64_t e = fill[(size_t)kt]++;
        q_tiles[e] = (int32_t)qt;
        kinds[e] = kind;
    });
    // processing order: most entries first (a k-tile's work grows with the q-tiles that see it)
    std::vector<int32_t> ord((size_t)nkt);
    std::iota(ord.begin(), ord.end(), 0);
    std::stable_sort(ord.begin(), ord.end(), [&](int32_t a, int32_t b) {
        return col_ptr[a + 1] - col_ptr[a] > col_ptr[b + 1] - col_ptr[b];
    });
    std::copy(ord.begin(), ord.end(), k_order);
    return PADOC_OK;
}

extern "C" padoc_status padoc_prefill_bwd_tile_shapes(padoc_dtype dtype, int32_t head_dim, int32_t *dq_q_tile,
                                                      int32_t *dq_k_tile, int32_t *dkv_q_tile, int32_t *dkv_k_tile)
{
    if (!dq_q_tile || !dq_k_tile || !dkv_q_tile || !dkv_k_tile) return PADOC_ERR_INVALID_ARGUMENT;
    const bool ok = (dtype == PADOC_DTYPE_BF16 && head_dim == 128) ||
                    (dtype == PADOC_DTYPE_F32 && (head_dim == 64 || head_dim == 128));
    if (!ok) return PADOC_ERR_UNSUPPORTED;
    *dq_q_tile = PADOC_BWD_DQ_Q_TILE;
    *dq_k_tile = PADOC_BWD_DQ_K_TILE;
    *dkv_q_tile = PADOC_BWD_DKV_Q_TILE;
    *dkv_k_tile = PADOC_BWD_DKV_K_TILE;
    return PADOC_OK;
}

// ------------------------------------------------------------------------------------------------
// Decode plan
// ------------------------------------------------------------------------------------------------

// Multiprocessor count of the current CUDA device, or 152 (one GB300) when none is visible; the
// device attribute is read once per device (a plan is built for every decode step).
int32_t padoc_default_ctas()
{
    constexpr int kMaxDevices = 64;
    static std::atomic<int32_t> cached[kMaxDevices];   // 0: not read yet
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return 152;
    }
    if (dev >= 0 && dev < kMaxDevices) {
        const int32_t c = cached[dev].load(std::memory_order_relaxed);
        if (c > 0) return c;
    }
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) {
        cudaGetLastError();
        n = 152;
    }
    if (dev >= 0 && dev < kMaxDevices) cached[dev].store(n, std::memory_order_relaxed);
    return n;
}

namespace {

int32_t choose_tc_ctas(const PlanParts &pp, const padoc_decode_config *cfg, int64_t total_w, int64_t max_piece,
                       int32_t split, int32_t psplit);
double warp_blocks_per_warp(const PlanParts &pp, const padoc_decode_config *cfg, int32_t min_rows);
int32_t warp_split_tokens(double blocks_per_warp);

padoc_status check_config(const padoc_decode_config *cfg)
{
    if (!cfg) return PADOC_ERR_INVALID_ARGUMENT;
    if (cfg->num_q_heads < 1 || cfg->num_kv_heads < 1 || cfg->num_q_heads % cfg->num_kv_heads != 0)
        return PADOC_ERR_INVALID_ARGUMENT;
    if (cfg->head_dim < 1 || cfg->block_size < 1) return PADOC_ERR_INVALID_ARGUMENT;
    if (cfg->block_size != 16) return PADOC_ERR_UNSUPPORTED;
    if (cfg->split_tokens < 0 || (cfg->split_tokens > 0 && cfg->split_tokens % cfg->block_size != 0))
        return PADOC_ERR_INVALID_ARGUMENT;
    if (cfg->tc_ctas < 0 || cfg->warp_ctas < 0) return PADOC_ERR_INVALID_ARGUMENT;
    return PADOC_OK;
}

// Streams of the pages (each page's branches, then its layout stream when cfg->layout_streams).
padoc_status streams_of_pages(const padoc_page *pages, int32_t num_pages, const padoc_decode_config *cfg,
                              PlanParts &pp)
{
    if (num_pages < 0 || (num_pages > 0 && !pages)) return PADOC_ERR_INVALID_ARGUMENT;
    int64_t ns = 0;
    for (int32_t p = 0; p < num_pages; ++p) ns += std::max(pages[p].num_branches, 0) + (cfg->layout_streams ? 1 : 0);
    pp.streams.reserve((size_t)ns);
    pp.page_len.reserve((size_t)num_pages);
    pp.page_first_stream.reserve((size_t)num_pages);
    pp.page_num_streams.reserve((size_t)num_pages);
    for (int32_t p = 0; p < num_pages; ++p) {
        const padoc_page &pg = pages[p];
        if (pg.prefix_len < 0 || pg.layout_len < 0 || pg.num_branches < 0) return PADOC_ERR_INVALID_ARGUMENT;
        if (pg.num_branches > 0 && (!pg.fork_offset || !pg.branch_len)) return PADOC_ERR_INVALID_ARGUMENT;
        const int64_t plen = (int64_t)pg.prefix_len + pg.layout_len;
        if (plen >= (int64_t)1 << 30) return PADOC_ERR_INVALID_ARGUMENT;
        pp.page_len.push_back((int32_t)plen);
        pp.page_first_stream.push_back((int32_t)pp.streams.size());
        for (int32_t k = 0; k < pg.num_branches; ++k) {
            if (pg.fork_offset[k] < 0 || pg.fork_offset[k] > pg.layout_len) return PADOC_ERR_INVALID_ARGUMENT;
            if (pg.branch_len[k] < 1 || pg.branch_len[k] >= (1 << 30)) return PADOC_ERR_INVALID_ARGUMENT;
            pp.streams.push_back({p, pg.prefix_len + pg.fork_offset[k], pg.branch_len[k]});
        }
        if (cfg->layout_streams) {
            if (plen < 1) return PADOC_ERR_INVALID_ARGUMENT;  // a layout stream decodes its newest token
            pp.streams.push_back({p, (int32_t)plen, 0});
        }
        pp.page_num_streams.push_back((int32_t)pp.streams.size() - pp.page_first_stream.back());
    }
    return PADOC_OK;
}

// An explicit stream list: page_len[p] shared-stream tokens of page p, streams grouped by page in
// ascending page order, each cutting the page's shared stream at shared_len <= page_len.
padoc_status streams_of_list(const int32_t *page_len, int32_t num_pages, const padoc_stream_desc *streams,
                             int32_t num_streams, PlanParts &pp)
{
    if (num_pages < 0 || num_streams < 0 || (num_pages > 0 && !page_len) || (num_streams > 0 && !streams))
        return PADOC_ERR_INVALID_ARGUMENT;
    for (int32_t p = 0; p < num_pages; ++p) {
        if (page_len[p] < 0 || page_len[p] >= (1 << 30)) return PADOC_ERR_INVALID_ARGUMENT;
        pp.page_len.push_back(page_len[p]);
    }
    pp.page_first_stream.assign(num_pages, 0);
    pp.page_num_streams.assign(num_pages, 0);
    int32_t prev = 0;
    for (int32_t s = 0; s < num_streams; ++s) {
        const padoc_stream_desc &d = streams[s];
        if (d.page < prev || d.page >= num_pages) return PADOC_ERR_INVALID_ARGUMENT;  // grouped, ascending
        if (d.shared_len < 0 || d.shared_len > page_len[d.page]) return PADOC_ERR_INVALID_ARGUMENT;
        if (d.private_len < 0 || d.private_len >= (1 << 30)) return PADOC_ERR_INVALID_ARGUMENT;
        if (pp.page_num_streams[d.page]++ == 0) pp.page_first_stream[d.page] = s;
        prev = d.page;
        pp.streams.push_back({d.page, d.shared_len, d.private_len});
    }
    for (int32_t p = 0; p < num_pages; ++p)
        if (pp.page_num_streams[p] == 0) pp.page_first_stream[p] = p > 0 ? pp.page_first_stream[p - 1] + pp.page_num_streams[p - 1] : 0;
    return PADOC_OK;
}

// A chunked prefill: each chunk's tokens become consecutive streams. A branch chunk (private_start
// >= 0) of n tokens: token i sees the page's shared stream before shared_len and its private rows
// [0, private_start + i + 1). A shared-stream chunk (private_start = -1): token i is shared row
// shared_len + i and sees the shared rows up to and including itself.
padoc_status streams_of_chunks(const int32_t *page_len, int32_t num_pages, const padoc_prefill_chunk *chunks,
                               int32_t num_chunks, PlanParts &pp)
{
    if (num_pages < 0 || num_chunks < 0 || (num_pages > 0 && !page_len) || (num_chunks > 0 && !chunks))
        return PADOC_ERR_INVALID_ARGUMENT;
    std::vector<padoc_stream_desc> list;
    int32_t prev = 0;
    for (int32_t c = 0; c < num_chunks; ++c) {
        const padoc_prefill_chunk &k = chunks[c];
        if (k.page < prev || k.page >= num_pages || k.num_tokens < 1 || k.shared_len < 0 || k.private_start < -1)
            return PADOC_ERR_INVALID_ARGUMENT;
        const int32_t pl = page_len[k.page];
        if (pl < 0 || k.shared_len > pl) return PADOC_ERR_INVALID_ARGUMENT;
        if (k.private_start < 0 && (int64_t)k.shared_len + k.num_tokens > pl) return PADOC_ERR_INVALID_ARGUMENT;
        if (k.private_start >= 0 && (int64_t)k.private_start + k.num_tokens >= (1 << 30)) return PADOC_ERR_INVALID_ARGUMENT;
        if ((int64_t)list.size() + k.num_tokens >= (1 << 30)) return PADOC_ERR_INVALID_ARGUMENT;
        prev = k.page;
        pp.chunk_first.push_back((int32_t)list.size());
        pp.chunk_len.push_back(k.num_tokens);
        pp.chunk_private.push_back(k.private_start >= 0 ? 1 : 0);
        for (int32_t i = 0; i < k.num_tokens; ++i) {
            pp.chunk_of.push_back(c);
            if (k.private_start >= 0)
                list.push_back({k.page, k.shared_len, k.private_start + i + 1});
            else
                list.push_back({k.page, k.shared_len + i + 1, 0});
        }
    }
    return streams_of_list(page_len, num_pages, list.data(), (int32_t)list.size(), pp);
}

// The split-K work of a stream list (pp.streams, page_len, page_first_stream, page_num_streams).
padoc_status build_work(int32_t num_pages, const padoc_decode_config *cfg, PlanParts &pp)
{
    const int32_t bs = cfg->block_size;
    const bool chunked = !pp.chunk_of.empty();
    // Pages whose shared stream the tensor cores read (once for all the page's streams): those of at
    // least PADOC_TC_MIN_ROWS rows (streams x query heads), and in a decode step with much warp work
    // those of at least PADOC_TC_MIN_ROWS_BUSY: there the warp path, which reads a page's shared
    // stream once per stream, would read it two to seven times (measured on GB300 over the decoding
    // loop's steps of 200-300 and of about 76 streams: 41.6 -> 31.5 and 33.3 -> 27.1 us per step)
    const double bpw = warp_blocks_per_warp(pp, cfg, PADOC_TC_MIN_ROWS);
    const int32_t min_rows = !chunked && bpw >= PADOC_TC_BUSY_BLOCKS ? PADOC_TC_MIN_ROWS_BUSY : PADOC_TC_MIN_ROWS;
    pp.tc_min_rows = min_rows;
    const int32_t auto_split = cfg->split_tokens > 0 ? 0 : warp_split_tokens(bpw);
    const int32_t split = cfg->split_tokens > 0 ? std::min(cfg->split_tokens, PADOC_WARP_MAX_ITEM_TOKENS) : auto_split;
    const int32_t psplit = cfg->split_tokens > 0 ? PADOC_PRIVATE_SPLIT_TOKENS : auto_split;
    const int32_t group = cfg->num_q_heads / cfg->num_kv_heads;

    for (int32_t p = 0; p < num_pages; ++p) {
        const int64_t plen = pp.page_len[p];
        pp.max_page_blocks = std::max<int32_t>(pp.max_page_blocks, (int32_t)((plen + bs - 1) / bs));
        if (pp.page_num_streams[p] > 0) pp.kv_tokens += plen;
    }
    const int32_t S = (int32_t)pp.streams.size();
    for (const PlanStream &s : pp.streams) {
        if (s.shared_len + s.private_len < 1) return PADOC_ERR_INVALID_ARGUMENT;
        pp.max_stream_blocks = std::max<int32_t>(pp.max_stream_blocks, (s.private_len + bs - 1) / bs);
        pp.kv_tokens += s.private_len;
    }

    // ---- tensor-core work: stream-K over the concatenated shared-stream tiles ----------------
    // A segment is one (KV head, page, group of <= 32 streams) with the tiles of the shared stream
    // the group can see. The segments are laid end to end and cut into one contiguous range per CTA
    // (a tile weighs PADOC_TC_WEIGHT_2M for a group of two M-tiles and PADOC_TC_WEIGHT_1M for one);
    // a range becomes the pieces where it overlaps segments.
    // A chunked prefill groups streams within a chunk only, and a group of a chunk whose tokens have
    // private rows and are many enough continues its segment over those rows (PADOC_ITEM_PRIVATE_TC,
    // through the chunk's first token's block-table row): the shared tiles, then the private ones,
    // one sequence with one running softmax, so that a piece covering both writes one partial. A
    // piece that crosses from the shared to the private tiles becomes two items, the first flagged
    // PADOC_ITEM_CONT; every stream of a group receives the same items and partial-slot numbers.
    using Segment = PlanSegment;
    PlanScratch &sc = pp.scratch;
    std::vector<Segment> &segs = sc.segs;
    segs.clear();
    std::vector<uint8_t> &priv_tc = sc.priv_tc;
    priv_tc.assign(chunked ? (size_t)S : 0, 0);
    auto weight_of = [](int32_t nb) { return nb > PADOC_TC_ITEM_STREAMS / 2 ? PADOC_TC_WEIGHT_2M : PADOC_TC_WEIGHT_1M; };
    for (int32_t g = 0; g < cfg->num_kv_heads; ++g) {
        for (int32_t p = 0; p < num_pages; ++p) {
            const int32_t f0 = pp.page_first_stream[p], ns = pp.page_num_streams[p];
            if ((int64_t)ns * group < min_rows) continue;
            for (int32_t r = 0; r < ns;) {
                int32_t nb = std::min(PADOC_TC_ITEM_STREAMS, ns - r);
                if (chunked)
                    for (int32_t j = 1; j < nb; ++j)
                        if (pp.chunk_of[f0 + r + j] != pp.chunk_of[f0 + r] ||
                            (f0 + r + j - pp.chunk_first[pp.chunk_of[f0 + r + j]]) % PADOC_TC_ITEM_STREAMS == 0) {
                            nb = j;
                            break;
                        }
                int32_t vis = 0;
                for (int32_t st = f0 + r; st < f0 + r + nb; ++st) vis = std::max(vis, pp.streams[st].shared_len);
                Segment sg{PADOC_ITEM_SHARED_TC | (chunked && nb < ns ? PADOC_ITEM_REREAD : 0), g, p, f0 + r, nb, vis,
                           (vis + PADOC_TC_TILE_TOKENS - 1) / PADOC_TC_TILE_TOKENS, weight_of(nb), 0, 0, 0, 0};
                if (chunked) {
                    // a group of a chunk with private rows on the tensor cores continues over them
                    const int32_t c = pp.chunk_of[f0 + r], first = pp.chunk_first[c], len = pp.chunk_len[c];
                    if (pp.chunk_private[c] && (int64_t)len * group >= min_rows) {
                        const int32_t vis2 = pp.streams[f0 + r + nb - 1].private_len;   // increasing within a chunk
                        for (int32_t st = f0 + r; st < f0 + r + nb; ++st) priv_tc[st] = 1;
                        sg.kind2 = PADOC_ITEM_PRIVATE_TC | (nb < len ? PADOC_ITEM_REREAD : 0);
                        sg.p2 = first;
                        sg.vis2 = vis2;
                        sg.ntiles2 = (vis2 + PADOC_TC_TILE_TOKENS - 1) / PADOC_TC_TILE_TOKENS;
                    }
                }
                if (sg.ntiles + sg.ntiles2 > 0) segs.push_back(sg);
                r += nb;
            }
        }
    }
    const int32_t Hkv = cfg->num_kv_heads;
    std::vector<int32_t> &cnt = sc.cnt;   // partial slots handed out per (stream, KV head)
    cnt.assign((size_t)S * Hkv, 0);
    std::vector<padoc_item> &tc_items = sc.tc_items;
    tc_items.clear();
    tc_items.reserve(segs.size() * 2 + 64);
    // CTA loads count every piece's own cost too (its epilogue, and the query reload before it):
    // the smallest bound T for which a greedy walk along the sequences needs at most `want` CTAs
    // is found by bisection, then the walk is made once more to emit the pieces.
    auto piece_cost = [&](const Segment &sg) -> int64_t {
        return (sg.weight == PADOC_TC_WEIGHT_2M ? PADOC_TC_PIECE_COST_2M : PADOC_TC_PIECE_COST_1M) +
               (chunked ? PADOC_TC_PIECE_EXTRA_CHUNK : 0);
    };
    int64_t max_piece = 0;
    int64_t total_w = 0, max_w = 0;
    for (const Segment &sg : segs) {
        total_w += (int64_t)(sg.ntiles + sg.ntiles2) * sg.weight + piece_cost(sg);
        max_piece = std::max(max_piece, piece_cost(sg));
        max_w = std::max<int64_t>(max_w, sg.weight);
    }
    std::vector<int64_t> &tc_load = sc.tc_load;   // planned load of each tensor-core CTA (emitting walk)
    tc_load.clear();
    auto walk = [&](int64_t T, bool emit) {
        int64_t used = 0, load = 0;
        for (const Segment &sg : segs) {
            int32_t t = 0;
            const int32_t ntot = sg.ntiles + sg.ntiles2;
            while (t < ntot) {
                const int64_t piece_w = piece_cost(sg);
                int64_t room = used > 0 ? (T - load - piece_w) / sg.weight : 0;
                if (room < 1) {   // close the current CTA, open the next
                    if (emit) {
                        if (used > 0) tc_load.push_back(load);
                        pp.cta_ptr.push_back((int32_t)tc_items.size());
                    }
                    ++used;
                    load = 0;
                    room = std::max<int64_t>(1, (T - piece_w) / sg.weight);
                }
                const int32_t t1 = (int32_t)std::min<int64_t>(ntot, t + room);
                load += piece_w + (int64_t)(t1 - t) * sg.weight;
                if (emit) {
                    // one partial slot per piece; a piece over shared and private tiles is two items
                    const int32_t slot = cnt[(size_t)sg.first * Hkv + sg.g];
                    for (int32_t st = sg.first; st < sg.first + sg.ns; ++st) ++cnt[(size_t)st * Hkv + sg.g];
                    if (t < sg.ntiles) {
                        const int32_t e = std::min(t1, sg.ntiles);
                        const int32_t tb = t * PADOC_TC_TILE_TOKENS, te = std::min(sg.vis, e * PADOC_TC_TILE_TOKENS);
                        tc_items.push_back({sg.kind | (t1 > sg.ntiles ? PADOC_ITEM_CONT : 0), sg.p, sg.g, tb, te,
                                            sg.first, sg.ns, slot});
                    }
                    if (t1 > sg.ntiles) {
                        const int32_t b = std::max(t, sg.ntiles) - sg.ntiles, e = t1 - sg.ntiles;
                        const int32_t tb = b * PADOC_TC_TILE_TOKENS, te = std::min(sg.vis2, e * PADOC_TC_TILE_TOKENS);
                        tc_items.push_back({sg.kind2, sg.p2, sg.g, tb, te, sg.first, sg.ns, slot});
                    }
                }
                t = t1;
            }
        }
        if (emit && used > 0) tc_load.push_back(load);
        return used;
    };
    int32_t ctas = 0;
    if (!segs.empty()) {
        const int64_t want = cfg->tc_ctas > 0 ? cfg->tc_ctas : choose_tc_ctas(pp, cfg, total_w, max_piece, split, psplit);
        // Every CTA's load stays within T (T >= max_w + max_piece), so T below total_w / want needs
        // more than `want` CTAs: that is a lower bound. A CTA is closed only once less than a piece
        // and a tile fit, and cutting adds at most one piece per CTA, so T = total_w / (want - 1) +
        // 2 max_piece + max_w fits in `want`; it is checked, with the one-CTA bound behind it.
        // The search depends only on `want` and each segment's tile count and weight (the rest follows
        // from them); a caller that plans step after step with the same parts (the decoding loop's
        // scheduler) often repeats them, and then the last bound is taken as it is.
        std::vector<int64_t> &key = sc.bound_key;
        key.clear();
        key.push_back(want);
        key.push_back(chunked ? 1 : 0);
        for (const Segment &sg : segs) key.push_back(((int64_t)(sg.ntiles + sg.ntiles2) << 8) | sg.weight);
        int64_t lo;
        if (sc.bound >= 0 && key == sc.last_bound_key) {
            lo = sc.bound;
        } else {
            lo = std::max<int64_t>(max_w + max_piece, (total_w + want - 1) / want);
            int64_t hi = (want > 1 ? (total_w + want - 2) / (want - 1) : total_w) + 2 * max_piece + max_w + 1;
            if (hi < lo || walk(hi, false) > want) hi = std::max(lo, total_w + max_w);   // walk(total_w + max_w) needs one CTA
            while (lo < hi) {
                const int64_t mid = lo + (hi - lo) / 2;
                if (walk(mid, false) <= want) hi = mid; else lo = mid + 1;
            }
            sc.last_bound_key.swap(key);
            sc.bound = lo;
        }
        ctas = (int32_t)walk(lo, true);
        pp.cta_ptr.push_back((int32_t)tc_items.size());
        // The CTAs in order of planned load, lightest first, so that they are predicted to end in
        // index order: warp CTA early + j then follows tensor-core CTA j's pieces in the decode grid,
        // and takes the SM of the j-th CTA to end in a warp grid of its own (the E4M3 pool), both
        // with the start the warp planning below gives it.
        std::vector<int32_t> &perm = sc.perm;
        perm.resize((size_t)ctas);
        std::iota(perm.begin(), perm.end(), 0);
        std::stable_sort(perm.begin(), perm.end(),
                         [&](int32_t a, int32_t b) { return tc_load[(size_t)a] < tc_load[(size_t)b]; });
        std::vector<padoc_item> &items_sorted = sc.items_sorted;
        items_sorted.clear();
        items_sorted.reserve(tc_items.size());
        std::vector<int32_t> &ptr_sorted = sc.ptr_sorted;
        ptr_sorted.assign(1, 0);
        std::vector<int64_t> &load_sorted = sc.load_sorted;
        load_sorted.clear();
        for (int32_t c : perm) {
            items_sorted.insert(items_sorted.end(), tc_items.begin() + pp.cta_ptr[(size_t)c],
                                tc_items.begin() + pp.cta_ptr[(size_t)c + 1]);
            ptr_sorted.push_back((int32_t)items_sorted.size());
            load_sorted.push_back(tc_load[(size_t)c]);
        }
        tc_items.swap(items_sorted);
        pp.cta_ptr.swap(ptr_sorted);
        tc_load.swap(load_sorted);
    }
    pp.tc_ctas = ctas;

    // ---- warp work: shared streams of sparse pages (per stream) and every private history ------
    std::vector<padoc_item> &warp_items = sc.warp_items;
    warp_items.clear();
    {
        int64_t n = 0;   // exact count, so the list is allocated once
        for (int32_t p = 0; p < num_pages; ++p) {
            const int32_t f0 = pp.page_first_stream[p], ns = pp.page_num_streams[p];
            if ((int64_t)ns * group >= min_rows) continue;
            for (int32_t st = f0; st < f0 + ns; ++st) n += (pp.streams[st].shared_len + split - 1) / split;
        }
        for (int32_t st = 0; st < S; ++st) n += (pp.streams[st].private_len + psplit - 1) / psplit + 1;
        warp_items.reserve((size_t)(n * Hkv));
    }
    for (int32_t g = 0; g < Hkv; ++g) {
        for (int32_t p = 0; p < num_pages; ++p) {
            const int32_t f0 = pp.page_first_stream[p], ns = pp.page_num_streams[p];
            if ((int64_t)ns * group >= min_rows) continue;
            for (int32_t st = f0; st < f0 + ns; ++st)
                for (int32_t tb = 0; tb < pp.streams[st].shared_len; tb += split)
                    warp_items.push_back({PADOC_ITEM_SHARED, p, g, tb, std::min(pp.streams[st].shared_len, tb + split),
                                          st, 1, cnt[(size_t)st * Hkv + g]++});
        }
        for (int32_t st = 0; st < S; ++st) {
            if (chunked && priv_tc[st]) continue;   // the chunk's private rows go to the tensor cores
            const int32_t L = pp.streams[st].private_len;
            for (int32_t tb = 0; tb < L; tb += psplit)
                warp_items.push_back({PADOC_ITEM_PRIVATE, st, g, tb, std::min(L, tb + psplit), st, 1,
                                      cnt[(size_t)st * Hkv + g]++});
        }
    }
    // a (stream, KV head) with nothing visible at all still gets one (empty) partial
    for (int32_t st = 0; st < S; ++st)
        for (int32_t g = 0; g < Hkv; ++g)
            if (cnt[(size_t)st * Hkv + g] == 0) {
                warp_items.push_back({PADOC_ITEM_SHARED, pp.streams[st].page, g, 0, 0, st, 1, 0});
                cnt[(size_t)st * Hkv + g] = 1;
            }
    pp.slot_ptr.assign((size_t)S * Hkv + 1, 0);
    for (size_t i = 0; i < (size_t)S * Hkv; ++i) pp.slot_ptr[i + 1] = pp.slot_ptr[i] + cnt[i];
    // A tensor-core item whose every stream has this one partial for its KV head (a chunked
    // prefill's group whose pieces stay on one CTA) writes their outputs itself; only the other
    // (stream, KV head) keys go to the merge.
    {
        std::vector<uint8_t> &direct = sc.direct;
        direct.assign((size_t)S * Hkv, 0);
        for (padoc_item &it : tc_items) {
            if (it.kind & PADOC_ITEM_CONT) continue;   // the next item of the chain writes
            bool sole = true;
            for (int32_t b = 0; sole && b < it.num_streams; ++b)
                sole = cnt[(size_t)(it.first_stream + b) * Hkv + it.kv_head] == 1;
            if (!sole) continue;
            it.kind |= PADOC_ITEM_SOLE;
            for (int32_t b = 0; b < it.num_streams; ++b) direct[(size_t)(it.first_stream + b) * Hkv + it.kv_head] = 1;
        }
        pp.merge_keys.clear();
        for (size_t i = 0; i < (size_t)S * Hkv; ++i)
            if (!direct[i]) pp.merge_keys.push_back((int32_t)i);
    }

    // The warp grid runs as one wave. Items are taken longest first (LPT; a counting sort on the
    // block count keeps ties in plan order) and each goes to the warp with the most capacity left
    // (below). Cost: 16-token blocks plus a fixed start-up cost per item.
    const int32_t nitems = (int32_t)warp_items.size();
    std::vector<int32_t> &cost = sc.cost, &order = sc.order;
    cost.resize((size_t)nitems);
    order.resize((size_t)nitems);
    int32_t maxb = 0;
    for (int32_t i = 0; i < nitems; ++i) {
        const int32_t nb = (warp_items[(size_t)i].tok_end - warp_items[(size_t)i].tok_begin + 15) / 16;
        cost[(size_t)i] = nb;
        maxb = std::max(maxb, nb);
    }
    {
        std::vector<int32_t> &first = sc.counts;   // first position of each block count, longest first
        first.assign((size_t)maxb + 2, 0);
        for (int32_t i = 0; i < nitems; ++i) ++first[(size_t)(maxb - cost[(size_t)i]) + 1];
        for (int32_t b = 0; b <= maxb; ++b) first[(size_t)b + 1] += first[(size_t)b];
        for (int32_t i = 0; i < nitems; ++i) order[(size_t)first[(size_t)(maxb - cost[(size_t)i])]++] = i;
    }
    for (int32_t i = 0; i < nitems; ++i) cost[(size_t)i] += PADOC_WARP_ITEM_COST;
    const int32_t wctas = (int32_t)std::min<int64_t>(cfg->warp_ctas > 0 ? cfg->warp_ctas : padoc_default_ctas(),
                                                     ((int64_t)nitems + PADOC_WARP_KERNEL_WARPS - 1) / PADOC_WARP_KERNEL_WARPS);
    const int32_t nwarps = (int32_t)std::min<int64_t>((int64_t)wctas * PADOC_WARP_KERNEL_WARPS, nitems);
    pp.warp_ptr.assign((size_t)nwarps + 1, 0);
    pp.num_tc_items = (int32_t)tc_items.size();
    pp.items.resize(tc_items.size() + (size_t)nitems);
    std::copy(tc_items.begin(), tc_items.end(), pp.items.begin());
    if (nwarps > 0) {
        // Warp CTAs start at different times (the fused grid's mapping is in plan_internal.h): the
        // first `early` of them on SMs the tensor-core CTAs leave free, soon after launch; warp CTA
        // early + j on tensor-core CTA j once its pieces end (predicted from its planned load). A
        // warp's share of the work is sized to the time it has: its capacity is its rate times
        // (T - its CTA's start - the time to its first block), with T such that the capacities add
        // up to the work. Taking items longest first, each to the warp with the most capacity left,
        // puts the longest items on the warps that start first. Without tensor-core work every warp
        // starts at once and the capacities are equal.
        // the warps of a CTA start together: start, rate and warp count per CTA
        std::vector<double> &start = sc.start, &rate = sc.rate;
        start.assign((size_t)wctas, 0.0);
        rate.assign((size_t)wctas, PADOC_WARP_RATE);
        std::vector<int32_t> &nw_of = sc.nw_of;
        nw_of.resize((size_t)wctas);
        for (int32_t c = 0; c < wctas; ++c)
            nw_of[(size_t)c] = std::min<int32_t>(PADOC_WARP_KERNEL_WARPS, nwarps - c * PADOC_WARP_KERNEL_WARPS);
        if (!tc_load.empty()) {
            const int32_t nsm = padoc_default_ctas(), ntc = (int32_t)tc_load.size();
            const int32_t early = padoc_fused_early_ctas(ntc, wctas, nsm);
            // early warp CTAs past the SM count (a warp_ctas above it) wait for a CTA to end
            const int32_t resident = std::min(early, std::max(0, nsm - ntc));
            std::vector<double> &tend = sc.tend;
            tend.resize(tc_load.size());
            double tmax = 0.0;
            for (size_t c = 0; c < tc_load.size(); ++c) {
                tend[c] = PADOC_TC_END_US0 + PADOC_TC_US_PER_UNIT * (double)tc_load[c];
                tmax = std::max(tmax, tend[c]);
            }
            for (int32_t c = 0; c < wctas; ++c) {
                if (c < resident) {
                    start[(size_t)c] = PADOC_WARP_EARLY_START_US;
                    rate[(size_t)c] = PADOC_WARP_EARLY_RATE;
                } else {
                    const double t0 = c < early ? tmax : tend[(size_t)(c - early)];
                    start[(size_t)c] = t0 + PADOC_WARP_SWITCH_US + PADOC_WARP_FIRST_US;
                }
            }
        }
        int64_t total = 0;
        for (int32_t i = 0; i < nitems; ++i) total += cost[(size_t)i];
        // T solves sum_c nw_c rate_c max(0, T - start_c) = total, which is piecewise linear in T:
        // walk the CTAs in order of start, adding each one's slope, until the line reaches total
        std::vector<int32_t> &by_start = sc.by_start;
        by_start.resize((size_t)wctas);
        std::iota(by_start.begin(), by_start.end(), 0);
        std::sort(by_start.begin(), by_start.end(), [&](int32_t x, int32_t y) { return start[(size_t)x] < start[(size_t)y]; });
        double T = 0.0, slope = 0.0, icpt = 0.0;   // capacity at T = slope * T - icpt
        for (size_t j = 0; j < by_start.size(); ++j) {
            const int32_t c = by_start[j];
            slope += nw_of[(size_t)c] * rate[(size_t)c];
            icpt += nw_of[(size_t)c] * rate[(size_t)c] * start[(size_t)c];
            T = (icpt + (double)total) / slope;
            if (j + 1 == by_start.size() || T <= start[(size_t)by_start[j + 1]]) break;
        }
        // Longest item first, each to the warp with the most capacity left (integer cost units). The
        // largest capacity left never grows, so the warps sit in FIFO buckets by capacity left and a
        // cursor walks down to the highest non-empty bucket (O(1) per item). A warp's capacity left
        // never falls more than one item below the largest, so the buckets start at -(longest
        // item + 2).
        int64_t max_cost = 0, max_room = 0;
        for (int32_t i = 0; i < nitems; ++i) max_cost = std::max<int64_t>(max_cost, cost[(size_t)i]);
        std::vector<int64_t> &room = sc.room;
        room.resize((size_t)nwarps);
        for (int32_t w = 0; w < nwarps; ++w) {
            const int32_t c = w / PADOC_WARP_KERNEL_WARPS;
            room[(size_t)w] = (int64_t)(rate[(size_t)c] * std::max(0.0, T - start[(size_t)c]));
            max_room = std::max(max_room, room[(size_t)w]);
        }
        const int64_t off = max_cost + 2, nbuckets = max_room + off + 1;
        std::vector<int32_t> &head = sc.head, &tail = sc.tail, &next = sc.next;
        head.assign((size_t)nbuckets, -1);
        tail.assign((size_t)nbuckets, -1);
        next.assign((size_t)nwarps, -1);
        auto push = [&](int32_t w) {
            const int64_t b = std::max<int64_t>(0, room[(size_t)w] + off);
            next[(size_t)w] = -1;
            if (tail[(size_t)b] < 0) head[(size_t)b] = w; else next[(size_t)tail[(size_t)b]] = w;
            tail[(size_t)b] = w;
        };
        for (int32_t w = 0; w < nwarps; ++w) push(w);
        std::vector<int32_t> &warp_of = sc.warp_of;
        warp_of.resize((size_t)nitems);
        int64_t cur = nbuckets - 1;
        for (int32_t k : order) {
            while (head[(size_t)cur] < 0) --cur;
            const int32_t w = head[(size_t)cur];
            head[(size_t)cur] = next[(size_t)w];
            if (head[(size_t)cur] < 0) tail[(size_t)cur] = -1;
            warp_of[(size_t)k] = w;
            ++pp.warp_ptr[(size_t)w + 1];
            room[(size_t)w] -= cost[(size_t)k];
            push(w);
        }
        for (int32_t w = 0; w < nwarps; ++w) pp.warp_ptr[(size_t)w + 1] += pp.warp_ptr[(size_t)w];
        std::vector<int32_t> &wpos = sc.wpos;
        wpos.assign(pp.warp_ptr.begin(), pp.warp_ptr.end() - 1);
        padoc_item *dst = pp.items.data() + tc_items.size();
        for (int32_t k : order) dst[wpos[(size_t)warp_of[(size_t)k]]++] = warp_items[(size_t)k];   // longest first per warp
    }
    pp.num_warps = nwarps;
    return PADOC_OK;
}

// How many SMs the tensor-core grid gets when the caller leaves it to the planner. Fewer tensor-core
// CTAs make that grid run longer but leave SMs to warp CTAs from the start, where they use the
// memory bandwidth the tensor-core CTAs (bound by their softmax and MMA chain) leave unused. With
// the timing model above, each candidate count n (the SM count, then down in steps of 8 to half of
// it) gets a predicted end of step: the tensor-core CTAs end on average at
// PADOC_TC_END_US0 + PADOC_TC_US_PER_UNIT * (total load / n + one piece) and the last of them
// PADOC_TC_END_SPREAD_US later, and the warp work, sized to each warp's start as in the planner
// (warp CTAs that follow a tensor-core CTA's pieces start at the average end), ends at T; the count whose
// later of the two ends is earliest wins (the larger count on a tie).
// Tokens per warp item when the caller leaves the split to the planner (shared-stream and private
// items alike): PADOC_DEFAULT_SPLIT_TOKENS, or shorter items when the warp work is small against the
// warp grid. A step of a decoding loop with few live streams is latency-bound: its time is the
// longest item's chain of 16-token blocks (each warp keeps three in flight) plus the merge, so
// shorter items (more partials to merge) finish sooner once there are fewer than
// PADOC_SPLIT_128_BLOCKS (PADOC_SPLIT_64_BLOCKS) 16-token blocks of warp work per warp (measured on
// GB300 over the serving batch's decoding loop: 20.2 -> 15.2 us per step at 1-2 live streams, 21.4
// -> 19.3 us at 17, while steps of 70 or more streams are fastest with 256).
// 16-token blocks of warp work per warp of the grid when the pages below min_rows rows (streams x
// query heads) read their shared streams on the warp path.
double warp_blocks_per_warp(const PlanParts &pp, const padoc_decode_config *cfg, int32_t min_rows)
{
    const int32_t group = cfg->num_q_heads / cfg->num_kv_heads, bs = cfg->block_size;
    int64_t blocks = 0;   // per KV head: sparse pages' shared rows of every stream, every private row
    for (size_t p = 0; p < pp.page_len.size(); ++p) {
        const int32_t f0 = pp.page_first_stream[p], ns = pp.page_num_streams[p];
        if ((int64_t)ns * group >= min_rows) continue;
        for (int32_t st = f0; st < f0 + ns; ++st) blocks += (pp.streams[(size_t)st].shared_len + bs - 1) / bs;
    }
    for (const PlanStream &st : pp.streams) blocks += (st.private_len + bs - 1) / bs;
    blocks *= cfg->num_kv_heads;
    const int64_t warps = (int64_t)(cfg->warp_ctas > 0 ? cfg->warp_ctas : padoc_default_ctas()) * PADOC_WARP_KERNEL_WARPS;
    return (double)blocks / (double)warps;
}

int32_t warp_split_tokens(double blocks_per_warp)
{
    if (blocks_per_warp < PADOC_SPLIT_64_BLOCKS) return 64;
    if (blocks_per_warp < PADOC_SPLIT_128_BLOCKS) return 128;
    return PADOC_DEFAULT_SPLIT_TOKENS;
}

int32_t choose_tc_ctas(const PlanParts &pp, const padoc_decode_config *cfg, int64_t total_w, int64_t max_piece,
                       int32_t split, int32_t psplit)
{
    const int32_t nsm = padoc_default_ctas();
    const int32_t group = cfg->num_q_heads / cfg->num_kv_heads;
    // the warp work: its items and their cost, as the planner will cut them
    int64_t wcost = 0, witems = 0;
    auto add = [&](int32_t len, int32_t step) {
        for (int32_t tb = 0; tb < len; tb += step) {
            wcost += (std::min(len, tb + step) - tb + 15) / 16 + PADOC_WARP_ITEM_COST;
            ++witems;
        }
    };
    for (int32_t g = 0; g < cfg->num_kv_heads; ++g) {
        for (size_t p = 0; p < pp.page_len.size(); ++p) {
            const int32_t f0 = pp.page_first_stream[p], ns = pp.page_num_streams[p];
            if ((int64_t)ns * group >= pp.tc_min_rows) continue;
            for (int32_t st = f0; st < f0 + ns; ++st) add(pp.streams[(size_t)st].shared_len, split);
        }
        for (const PlanStream &st : pp.streams) add(st.private_len, psplit);
    }
    const int64_t wctas = std::min<int64_t>(cfg->warp_ctas > 0 ? cfg->warp_ctas : nsm,
                                            (witems + PADOC_WARP_KERNEL_WARPS - 1) / PADOC_WARP_KERNEL_WARPS);
    if (wcost == 0 || wctas == 0) return nsm;
    int32_t best_n = nsm;
    double best = 1e300;
    for (int32_t n = nsm; n >= std::max(1, nsm / 2); n -= 8) {
        const double tc_end = PADOC_TC_END_US0 + PADOC_TC_US_PER_UNIT * ((double)total_w / n + (double)max_piece);
        const double ne = (double)std::min<int64_t>(std::max(0, nsm - n), wctas), nl = (double)wctas - ne;
        const double se = PADOC_WARP_EARLY_START_US, sl = tc_end + PADOC_WARP_SWITCH_US + PADOC_WARP_FIRST_US;
        const double ae = PADOC_WARP_KERNEL_WARPS * PADOC_WARP_EARLY_RATE * ne, al = PADOC_WARP_KERNEL_WARPS * PADOC_WARP_RATE * nl;
        // capacity at T: ae (T - se) + al max(0, T - sl) (se < sl); solve for T = the warp work
        double T = ae > 0 ? se + (double)wcost / ae : 1e300;
        if (T > sl) T = (ae * se + al * sl + (double)wcost) / (ae + al);
        const double end = std::max(tc_end + PADOC_TC_END_SPREAD_US, T);
        if (end < best - 1e-9) {
            best = end;
            best_n = n;
        }
    }
    return best_n;
}

}  // namespace

// int32 words of the plan blob: stream_page, shared_len, private_len [S], slot_ptr [S Hkv + 1],
// items [num_items][8], page_len [num_pages], cta_ptr [tc_ctas + 1], warp_ptr [num_warps + 1],
// merge_keys [num_merge_keys]
int64_t padoc_plan_blob_ints(const PlanParts &pp, int32_t num_pages, int32_t hkv)
{
    const int64_t S = (int64_t)pp.streams.size();
    return 3 * S + (S * hkv + 1) + (int64_t)pp.items.size() * PADOC_ITEM_INTS + num_pages + (int64_t)pp.cta_ptr.size() +
           (int64_t)pp.warp_ptr.size() + (int64_t)pp.merge_keys.size();
}

namespace {

padoc_status parts_of_pages(const padoc_page *pages, int32_t num_pages, const padoc_decode_config *cfg,
                           PlanParts &pp)
{
    pp.reset();
    padoc_status st = check_config(cfg);
    if (st == PADOC_OK) st = streams_of_pages(pages, num_pages, cfg, pp);
    if (st == PADOC_OK) st = build_work(num_pages, cfg, pp);
    return st;
}

}  // namespace

padoc_status padoc_plan_parts_of_list(const int32_t *page_len, int32_t num_pages, const padoc_stream_desc *streams,
                                      int32_t num_streams, const padoc_decode_config *cfg, PlanParts &pp)
{
    pp.reset();
    padoc_status st = check_config(cfg);
    if (st == PADOC_OK && cfg->layout_streams) st = PADOC_ERR_INVALID_ARGUMENT;  // the list names every stream
    if (st == PADOC_OK) st = streams_of_list(page_len, num_pages, streams, num_streams, pp);
    if (st == PADOC_OK) st = build_work(num_pages, cfg, pp);
    return st;
}

padoc_status padoc_plan_parts_of_chunks(const int32_t *page_len, int32_t num_pages, const padoc_prefill_chunk *chunks,
                                        int32_t num_chunks, const padoc_decode_config *cfg, PlanParts &pp)
{
    pp.reset();
    padoc_status st = check_config(cfg);
    if (st == PADOC_OK && cfg->layout_streams) st = PADOC_ERR_INVALID_ARGUMENT;
    if (st == PADOC_OK) st = streams_of_chunks(page_len, num_pages, chunks, num_chunks, pp);
    if (st == PADOC_OK) st = build_work(num_pages, cfg, pp);
    return st;
}

padoc_status padoc_plan_write_blob(const PlanParts &pp, int32_t num_pages, const padoc_decode_config *cfg, int32_t *plan,
                                   int64_t capacity_ints, padoc_decode_plan *info)
{
    const int64_t S = (int64_t)pp.streams.size();
    const int64_t need = padoc_plan_blob_ints(pp, num_pages, cfg->num_kv_heads);
    if (capacity_ints < need) return PADOC_ERR_CAPACITY;
    if (need > 0 && !plan) return PADOC_ERR_INVALID_ARGUMENT;
    std::memset(info, 0, sizeof(*info));
    info->cfg = *cfg;
    info->num_pages = num_pages;
    info->num_streams = (int32_t)S;
    info->num_items = (int32_t)pp.items.size();
    info->num_tc_items = pp.num_tc_items;
    info->tc_ctas = pp.tc_ctas;
    info->num_warps = pp.num_warps;
    info->num_slots = pp.slot_ptr.back();
    info->max_page_blocks = pp.max_page_blocks;
    info->max_stream_blocks = pp.max_stream_blocks;
    for (size_t i = 0; i + 1 < pp.slot_ptr.size(); ++i)
        info->max_stream_slots = std::max<int32_t>(info->max_stream_slots, pp.slot_ptr[i + 1] - pp.slot_ptr[i]);
    info->plan_ints = need;
    info->kv_tokens = pp.kv_tokens;
    int64_t o = 0;
    info->off_stream_page = o; o += S;
    info->off_shared_len = o; o += S;
    info->off_private_len = o; o += S;
    info->off_slot_ptr = o; o += (int64_t)pp.slot_ptr.size();
    info->off_items = o; o += (int64_t)pp.items.size() * PADOC_ITEM_INTS;
    info->off_page_len = o; o += num_pages;
    info->off_cta_ptr = o; o += (int64_t)pp.cta_ptr.size();
    info->off_warp_ptr = o; o += (int64_t)pp.warp_ptr.size();
    info->off_merge_keys = o; o += (int64_t)pp.merge_keys.size();
    info->num_merge_keys = (int32_t)pp.merge_keys.size();
    for (int64_t s = 0; s < S; ++s) {
        plan[info->off_stream_page + s] = pp.streams[s].page;
        plan[info->off_shared_len + s] = pp.streams[s].shared_len;
        plan[info->off_private_len + s] = pp.streams[s].private_len;
    }
    std::memcpy(plan + info->off_slot_ptr, pp.slot_ptr.data(), pp.slot_ptr.size() * sizeof(int32_t));
    std::memcpy(plan + info->off_items, pp.items.data(), pp.items.size() * sizeof(padoc_item));
    for (int32_t p = 0; p < num_pages; ++p) plan[info->off_page_len + p] = pp.page_len[p];
    if (!pp.cta_ptr.empty()) std::memcpy(plan + info->off_cta_ptr, pp.cta_ptr.data(), pp.cta_ptr.size() * sizeof(int32_t));
    std::memcpy(plan + info->off_warp_ptr, pp.warp_ptr.data(), pp.warp_ptr.size() * sizeof(int32_t));
    if (!pp.merge_keys.empty())
        std::memcpy(plan + info->off_merge_keys, pp.merge_keys.data(), pp.merge_keys.size() * sizeof(int32_t));
    return PADOC_OK;
}

extern "C" padoc_status padoc_decode_plan_size(const padoc_page *pages, int32_t num_pages,
                                               const padoc_decode_config *cfg, int64_t *plan_ints)
{
    if (!plan_ints) return PADOC_ERR_INVALID_ARGUMENT;
    PlanParts pp;
    padoc_status st = parts_of_pages(pages, num_pages, cfg, pp);
    if (st != PADOC_OK) return st;
    *plan_ints = padoc_plan_blob_ints(pp, num_pages, cfg->num_kv_heads);
    return PADOC_OK;
}

extern "C" padoc_status padoc_build_decode_plan(const padoc_page *pages, int32_t num_pages,
                                                const padoc_decode_config *cfg, int32_t *plan,
                                                int64_t capacity_ints, padoc_decode_plan *info)
{
    if (!info) return PADOC_ERR_INVALID_ARGUMENT;
    PlanParts pp;
    padoc_status st = parts_of_pages(pages, num_pages, cfg, pp);
    if (st != PADOC_OK) return st;
    return padoc_plan_write_blob(pp, num_pages, cfg, plan, capacity_ints, info);
}

extern "C" padoc_status padoc_decode_plan_size_streams(const int32_t *page_len, int32_t num_pages,
                                                       const padoc_stream_desc *streams, int32_t num_streams,
                                                       const padoc_decode_config *cfg, int64_t *plan_ints)
{
    if (!plan_ints) return PADOC_ERR_INVALID_ARGUMENT;
    PlanParts pp;
    padoc_status st = padoc_plan_parts_of_list(page_len, num_pages, streams, num_streams, cfg, pp);
    if (st != PADOC_OK) return st;
    *plan_ints = padoc_plan_blob_ints(pp, num_pages, cfg->num_kv_heads);
    return PADOC_OK;
}

extern "C" padoc_status padoc_build_decode_plan_streams(const int32_t *page_len, int32_t num_pages,
                                                        const padoc_stream_desc *streams, int32_t num_streams,
                                                        const padoc_decode_config *cfg, int32_t *plan,
                                                        int64_t capacity_ints, padoc_decode_plan *info)
{
    if (!info) return PADOC_ERR_INVALID_ARGUMENT;
    PlanParts pp;
    padoc_status st = padoc_plan_parts_of_list(page_len, num_pages, streams, num_streams, cfg, pp);
    if (st != PADOC_OK) return st;
    return padoc_plan_write_blob(pp, num_pages, cfg, plan, capacity_ints, info);
}

extern "C" padoc_status padoc_decode_workspace_size(const padoc_decode_plan *info, size_t *bytes)
{
    if (!info || !bytes) return PADOC_ERR_INVALID_ARGUMENT;
    *bytes = padoc_decode_workspace_bytes(info->num_slots, info->cfg.num_q_heads / info->cfg.num_kv_heads,
                                          info->cfg.head_dim);
    return PADOC_OK;
}

// Patches a decode plan for new private lengths (the decoding loop's steady state: every stream
// appends one token per step, nothing forks or retires). Each stream's work stays where it is; the
// private item that ends at a stream's old length (one per KV head) is extended to the new one,
// which is allowed while the item stays within PADOC_WARP_MAX_ITEM_TOKENS (the planner cuts private
// histories at PADOC_PRIVATE_SPLIT_TOKENS, which leaves that much room to grow). Anything else
// (a shorter length, a stream that had no private rows, an item past the limit, a chunked-prefill
// plan) asks for a new plan.
extern "C" padoc_status padoc_advance_decode_plan(int32_t *plan, padoc_decode_plan *info, const int32_t *private_len,
                                                  int32_t num_streams)
{
    if (!plan || !info || (num_streams > 0 && !private_len)) return PADOC_ERR_INVALID_ARGUMENT;
    if (num_streams != info->num_streams) return PADOC_ERR_INVALID_ARGUMENT;
    const int32_t S = info->num_streams;
    const int32_t Hkv = info->cfg.num_kv_heads;
    if (Hkv < 1 || info->num_items < info->num_tc_items || info->num_tc_items < 0) return PADOC_ERR_INVALID_ARGUMENT;
    int32_t *old_len = plan + info->off_private_len;
    padoc_item *items = reinterpret_cast<padoc_item *>(plan + info->off_items);
    int64_t grow = 0;
    int32_t max_blocks = info->max_stream_blocks;
    for (int32_t s = 0; s < S; ++s) {
        const int32_t n = private_len[s], o = old_len[s];
        if (n < o || n >= (1 << 30)) return PADOC_ERR_CAPACITY;
        if (n > o && o == 0) return PADOC_ERR_CAPACITY;   // no private item to extend
        grow += n - o;
        max_blocks = std::max(max_blocks, (n + info->cfg.block_size - 1) / info->cfg.block_size);
    }
    for (int32_t i = 0; i < info->num_tc_items; ++i)
        if (PADOC_ITEM_KIND(items[i].kind) == PADOC_ITEM_PRIVATE_TC) return PADOC_ERR_CAPACITY;
    if (grow == 0) return PADOC_OK;
    // the items to extend: a private item of stream s whose end is s's old length (checked first,
    // changed after, so that a refusal leaves the plan as it was)
    int64_t extended = 0;
    for (int32_t i = info->num_tc_items; i < info->num_items; ++i) {
        const padoc_item &it = items[i];
        if (it.kind != PADOC_ITEM_PRIVATE || it.index < 0 || it.index >= S) continue;
        const int32_t s = it.index;
        if (it.tok_end != old_len[s] || private_len[s] == old_len[s]) continue;
        if (private_len[s] - it.tok_begin > PADOC_WARP_MAX_ITEM_TOKENS) return PADOC_ERR_CAPACITY;
        ++extended;
    }
    int64_t want = 0;
    for (int32_t s = 0; s < S; ++s) want += (private_len[s] != old_len[s]) ? Hkv : 0;
    if (extended != want) return PADOC_ERR_CAPACITY;
    for (int32_t i = info->num_tc_items; i < info->num_items; ++i) {
        padoc_item &it = items[i];
        if (it.kind == PADOC_ITEM_PRIVATE && it.index >= 0 && it.index < S && it.tok_end == old_len[it.index])
            it.tok_end = private_len[it.index];
    }
    for (int32_t s = 0; s < S; ++s) old_len[s] = private_len[s];
    info->max_stream_blocks = max_blocks;
    info->kv_tokens += grow;
    return PADOC_OK;
}

extern "C" padoc_status padoc_chunk_prefill_plan_size(const int32_t *page_len, int32_t num_pages,
                                                      const padoc_prefill_chunk *chunks, int32_t num_chunks,
                                                      const padoc_decode_config *cfg, int64_t *plan_ints)
{
    if (!plan_ints) return PADOC_ERR_INVALID_ARGUMENT;
    PlanParts pp;
    padoc_status st = padoc_plan_parts_of_chunks(page_len, num_pages, chunks, num_chunks, cfg, pp);
    if (st != PADOC_OK) return st;
    *plan_ints = padoc_plan_blob_ints(pp, num_pages, cfg->num_kv_heads);
    return PADOC_OK;
}

extern "C" padoc_status padoc_build_chunk_prefill_plan(const int32_t *page_len, int32_t num_pages,
                                                       const padoc_prefill_chunk *chunks, int32_t num_chunks,
                                                       const padoc_decode_config *cfg, int32_t *plan,
                                                       int64_t capacity_ints, padoc_decode_plan *info)
{
    if (!info) return PADOC_ERR_INVALID_ARGUMENT;
    PlanParts pp;
    padoc_status st = padoc_plan_parts_of_chunks(page_len, num_pages, chunks, num_chunks, cfg, pp);
    if (st != PADOC_OK) return st;
    return padoc_plan_write_blob(pp, num_pages, cfg, plan, capacity_ints, info);
}

extern "C" padoc_status padoc_expand_chunk_table(const padoc_prefill_chunk *chunks, int32_t num_chunks,
                                                 const int32_t *chunk_table, int32_t chunk_stride,
                                                 int32_t *stream_table, int32_t stream_stride, int64_t capacity_rows)
{
    if (num_chunks < 0 || (num_chunks > 0 && (!chunks || !chunk_table || !stream_table)) || chunk_stride < 1 ||
        stream_stride < chunk_stride)
        return PADOC_ERR_INVALID_ARGUMENT;
    int64_t rows = 0;
    for (int32_t c = 0; c < num_chunks; ++c) {
        if (chunks[c].num_tokens < 1) return PADOC_ERR_INVALID_ARGUMENT;
        rows += chunks[c].num_tokens;
    }
    if (rows > capacity_rows) return PADOC_ERR_CAPACITY;
    int64_t r = 0;
    for (int32_t c = 0; c < num_chunks; ++c)
        for (int32_t i = 0; i < chunks[c].num_tokens; ++i, ++r) {
            int32_t *dst = stream_table + r * stream_stride;
            std::memcpy(dst, chunk_table + (int64_t)c * chunk_stride, sizeof(int32_t) * (size_t)chunk_stride);
            std::fill(dst + chunk_stride, dst + stream_stride, -1);
        }
    return PADOC_OK;
}
