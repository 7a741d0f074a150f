// plan.cpp -- C1: ancestor descriptors, prefill tile map and decode plan (host, integer only).
//
// The visibility rule is the packed form of the ancestor sets (Sec. 3.2; App. C.1): within a page
// [X | layout | Y_1..Y_N], a prefix or layout token q sees [page_begin, q]; a branch token of Y_k
// sees [page_begin, page_begin + P + f_k) and [ybase_k, q]. Everything here is exact integer
// arithmetic; outputs are bit-exact and canonical (see padoc_attn.h).
#include <algorithm>
#include <cstdint>
#include <cstring>
#include <numeric>
#include <vector>

#include "padoc_attn.h"
#include "plan_internal.h"

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

// ------------------------------------------------------------------------------------------------
// Decode plan
// ------------------------------------------------------------------------------------------------

namespace {

struct Stream { int32_t page, shared_len, private_len; };

struct PlanParts {
    std::vector<Stream> streams;
    std::vector<int32_t> page_len, page_first_stream, page_num_streams;
    std::vector<int32_t> slot_ptr;
    std::vector<padoc_item> items;
    int32_t num_tc_items = 0;
    int32_t max_page_blocks = 0, max_stream_blocks = 0;
    int64_t kv_tokens = 0;
};

padoc_status build_parts(const padoc_page *pages, int32_t num_pages, const padoc_decode_config *cfg, PlanParts &pp)
{
    if (!cfg) return PADOC_ERR_INVALID_ARGUMENT;
    if (num_pages < 0 || (num_pages > 0 && !pages)) return PADOC_ERR_INVALID_ARGUMENT;
    if (cfg->num_q_heads < 1 || cfg->num_kv_heads < 1 || cfg->num_q_heads % cfg->num_kv_heads != 0)
        return PADOC_ERR_INVALID_ARGUMENT;
    if (cfg->head_dim < 1 || cfg->block_size < 1) return PADOC_ERR_INVALID_ARGUMENT;
    if (cfg->block_size != 16) return PADOC_ERR_UNSUPPORTED;
    if (cfg->split_tokens < 0 || (cfg->split_tokens > 0 && cfg->split_tokens % cfg->block_size != 0))
        return PADOC_ERR_INVALID_ARGUMENT;
    const int32_t bs = cfg->block_size;
    const int32_t split = std::min(cfg->split_tokens > 0 ? cfg->split_tokens : PADOC_DEFAULT_SPLIT_TOKENS,
                                   PADOC_TC_MAX_ITEM_TOKENS);
    const int32_t psplit = PADOC_PRIVATE_SPLIT_TOKENS;
    const int32_t group = cfg->num_q_heads / cfg->num_kv_heads;

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
        pp.max_page_blocks = std::max<int32_t>(pp.max_page_blocks, (int32_t)((plen + bs - 1) / bs));
        if (pp.page_num_streams.back() > 0) pp.kv_tokens += plen;
    }
    const int32_t S = (int32_t)pp.streams.size();
    for (const Stream &s : pp.streams) {
        if (s.shared_len + s.private_len < 1) return PADOC_ERR_INVALID_ARGUMENT;
        pp.max_stream_blocks = std::max<int32_t>(pp.max_stream_blocks, (s.private_len + bs - 1) / bs);
        pp.kv_tokens += s.private_len;
    }

    // split-K slots: shared splits of the stream's page, then its private splits
    std::vector<int32_t> page_splits(num_pages);
    for (int32_t p = 0; p < num_pages; ++p) {
        // only the part of the stream some stream of the page can see needs reading
        int32_t vis = 0;
        for (int32_t s = pp.page_first_stream[p]; s < pp.page_first_stream[p] + pp.page_num_streams[p]; ++s)
            vis = std::max(vis, pp.streams[s].shared_len);
        page_splits[p] = (vis + split - 1) / split;
    }
    pp.slot_ptr.assign((size_t)S + 1, 0);
    for (int32_t s = 0; s < S; ++s) {
        const int32_t np = page_splits[pp.streams[s].page];
        const int32_t nv = (pp.streams[s].private_len + psplit - 1) / psplit;
        pp.slot_ptr[s + 1] = pp.slot_ptr[s] + np + nv;
    }

    // work items, one set per KV head: tensor-core items first, then warp items
    std::vector<padoc_item> tc_items, warp_items;
    for (int32_t g = 0; g < cfg->num_kv_heads; ++g) {
        for (int32_t p = 0; p < num_pages; ++p) {
            const int32_t f0 = pp.page_first_stream[p], ns = pp.page_num_streams[p];
            int32_t vis = 0;
            for (int32_t s = f0; s < f0 + ns; ++s) vis = std::max(vis, pp.streams[s].shared_len);
            const bool use_tc = (int64_t)ns * group >= PADOC_TC_MIN_ROWS;
            for (int32_t j = 0; j < page_splits[p]; ++j) {
                const int32_t tb = j * split, te = std::min(vis, tb + split);
                if (use_tc) {
                    for (int32_t r = 0; r < ns; r += PADOC_TC_ITEM_STREAMS)
                        tc_items.push_back({PADOC_ITEM_SHARED_TC, p, g, tb, te, f0 + r,
                                            std::min(PADOC_TC_ITEM_STREAMS, ns - r), j});
                } else {
                    for (int32_t s = f0; s < f0 + ns; ++s) {
                        const int32_t tes = std::min(te, pp.streams[s].shared_len);
                        if (tes <= tb) {
                            // nothing of this split is visible to the stream: an empty partial
                            warp_items.push_back({PADOC_ITEM_SHARED, p, g, tb, tb, s, 1, j});
                        } else {
                            warp_items.push_back({PADOC_ITEM_SHARED, p, g, tb, tes, s, 1, j});
                        }
                    }
                }
            }
        }
        for (int32_t s = 0; s < S; ++s) {
            const int32_t np = page_splits[pp.streams[s].page];
            const int32_t L = pp.streams[s].private_len;
            for (int32_t tb = 0, i = 0; tb < L; tb += psplit, ++i)
                warp_items.push_back({PADOC_ITEM_PRIVATE, s, g, tb, std::min(L, tb + psplit), s, 1, np + i});
        }
    }
    // longest items first (LPT order) within each kernel's list, ties by position for determinism
    auto longer = [](const padoc_item &a, const padoc_item &b) {
        return (int64_t)(a.tok_end - a.tok_begin) * (a.num_streams + 15) > (int64_t)(b.tok_end - b.tok_begin) * (b.num_streams + 15);
    };
    std::stable_sort(tc_items.begin(), tc_items.end(), longer);
    std::stable_sort(warp_items.begin(), warp_items.end(), longer);
    pp.num_tc_items = (int32_t)tc_items.size();
    pp.items = tc_items;
    pp.items.insert(pp.items.end(), warp_items.begin(), warp_items.end());
    return PADOC_OK;
}

}  // namespace

extern "C" padoc_status padoc_decode_plan_size(const padoc_page *pages, int32_t num_pages,
                                               const padoc_decode_config *cfg, int64_t *plan_ints)
{
    if (!plan_ints) return PADOC_ERR_INVALID_ARGUMENT;
    PlanParts pp;
    padoc_status st = build_parts(pages, num_pages, cfg, pp);
    if (st != PADOC_OK) return st;
    const int64_t S = (int64_t)pp.streams.size();
    *plan_ints = 3 * S + (S + 1) + (int64_t)pp.items.size() * PADOC_ITEM_INTS + num_pages;
    return PADOC_OK;
}

extern "C" padoc_status padoc_build_decode_plan(const padoc_page *pages, int32_t num_pages,
                                                const padoc_decode_config *cfg, int32_t *plan,
                                                int64_t capacity_ints, padoc_decode_plan *info)
{
    if (!info) return PADOC_ERR_INVALID_ARGUMENT;
    PlanParts pp;
    padoc_status st = build_parts(pages, num_pages, cfg, pp);
    if (st != PADOC_OK) return st;
    const int64_t S = (int64_t)pp.streams.size();
    const int64_t need = 3 * S + (S + 1) + (int64_t)pp.items.size() * PADOC_ITEM_INTS + num_pages;
    if (capacity_ints < need) return PADOC_ERR_CAPACITY;
    if (need > 0 && !plan) return PADOC_ERR_INVALID_ARGUMENT;
    std::memset(info, 0, sizeof(*info));
    info->cfg = *cfg;
    info->num_pages = num_pages;
    info->num_streams = (int32_t)S;
    info->num_items = (int32_t)pp.items.size();
    info->num_tc_items = pp.num_tc_items;
    info->num_slots = pp.slot_ptr.back();
    info->max_page_blocks = pp.max_page_blocks;
    info->max_stream_blocks = pp.max_stream_blocks;
    for (int64_t st = 0; st < S; ++st)
        info->max_stream_slots = std::max<int32_t>(info->max_stream_slots, pp.slot_ptr[st + 1] - pp.slot_ptr[st]);
    info->plan_ints = need;
    info->kv_tokens = pp.kv_tokens;
    int64_t o = 0;
    info->off_stream_page = o; o += S;
    info->off_shared_len = o; o += S;
    info->off_private_len = o; o += S;
    info->off_slot_ptr = o; o += S + 1;
    info->off_items = o; o += (int64_t)pp.items.size() * PADOC_ITEM_INTS;
    info->off_page_len = o; o += num_pages;
    for (int64_t s = 0; s < S; ++s) {
        plan[info->off_stream_page + s] = pp.streams[s].page;
        plan[info->off_shared_len + s] = pp.streams[s].shared_len;
        plan[info->off_private_len + s] = pp.streams[s].private_len;
    }
    for (int64_t s = 0; s <= S; ++s) plan[info->off_slot_ptr + s] = pp.slot_ptr[s];
    std::memcpy(plan + info->off_items, pp.items.data(), pp.items.size() * sizeof(padoc_item));
    for (int32_t p = 0; p < num_pages; ++p) plan[info->off_page_len + p] = pp.page_len[p];
    return PADOC_OK;
}

extern "C" padoc_status padoc_decode_workspace_size(const padoc_decode_plan *info, size_t *bytes)
{
    if (!info || !bytes) return PADOC_ERR_INVALID_ARGUMENT;
    *bytes = padoc_decode_workspace_bytes(info->num_slots, info->cfg.num_q_heads, info->cfg.head_dim);
    return PADOC_OK;
}
