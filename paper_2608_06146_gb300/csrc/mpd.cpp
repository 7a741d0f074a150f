// mpd.cpp -- Algorithm 1 (App. E.1): host-side scheduler of the masked parallel decoding loop over
// the paged KV cache (C5).
//
// The logical state of App. E.1 is a cache of positions and a mask row per live stream. Here the
// cache is the block pool and a row is two numbers: the stream's cutoff on its page's shared stream
// (prefix X, then the layout stream's tokens in the order it appended them) and its private length.
// A step appends one input per live stream (M <- [M I_C]): the layout stream's input extends the
// shared stream, so every later fork sees it; a branch's input extends its own private rows, which
// no other stream can reach. A fork copies the layout stream's row before its boundary output is
// appended, which is the shared stream's current length. Retiring removes the row and returns the
// stream's private blocks; a page's shared blocks return once its last stream has retired.
#include <algorithm>
#include <climits>
#include <cstdint>
#include <cstring>
#include <deque>
#include <new>
#include <vector>

#include <cuda_runtime.h>

#include "padoc_attn.h"
#include "plan_build.h"

namespace {

struct MpdStream {
    int32_t page;                  // page id
    int32_t cutoff;                // branch: shared-stream cutoff, fixed at the fork
    int32_t priv_len;              // branch: private rows in the cache
    bool layout;
    bool live;
    std::vector<int32_t> blocks;   // branch: private blocks
};

struct MpdPage {
    int32_t shared_len;            // shared-stream tokens in the cache (prefix + layout tokens)
    int32_t layout_stream;         // id of the live layout stream, or -1
    std::vector<int32_t> blocks;   // shared-stream blocks
    std::vector<int32_t> branches; // live branch ids in fork order
};

}  // namespace

struct padoc_mpd {
    int32_t bs = 16;
    int32_t num_blocks = 0;
    std::deque<int32_t> free_blocks;
    std::vector<MpdPage> pages;        // by page id
    std::vector<int32_t> live_pages;   // page ids in admission order
    std::vector<MpdStream> streams;    // by stream id
    bool in_step = false;
    std::vector<int32_t> step_streams; // stream ids in step order
    std::vector<int32_t> scratch_len;  // padoc_mpd_prepare_step: the step's page lengths and streams
    std::vector<padoc_stream_desc> scratch_streams;
    PlanParts plan_parts;              // the step's plan (kept: its arrays are reused step after step)
};

namespace {

int32_t take_block(padoc_mpd *m)
{
    const int32_t b = m->free_blocks.front();
    m->free_blocks.pop_front();
    return b;
}

void give_blocks(padoc_mpd *m, std::vector<int32_t> &blocks)
{
    for (int32_t b : blocks) m->free_blocks.push_back(b);
    std::vector<int32_t>().swap(blocks);
}

int32_t new_stream(padoc_mpd *m, int32_t page, bool layout, int32_t cutoff)
{
    MpdStream s;
    s.page = page;
    s.cutoff = cutoff;
    s.priv_len = 0;
    s.layout = layout;
    s.live = true;
    m->streams.push_back(std::move(s));
    return (int32_t)m->streams.size() - 1;
}

int32_t page_streams(const MpdPage &pg) { return (int32_t)pg.branches.size() + (pg.layout_stream >= 0 ? 1 : 0); }

}  // namespace

extern "C" padoc_status padoc_mpd_create(int32_t num_blocks, int32_t block_size, const int32_t *block_order,
                                         padoc_mpd **mpd)
{
    if (!mpd || num_blocks < 0 || block_size < 1) return PADOC_ERR_INVALID_ARGUMENT;
    if (block_size != 16) return PADOC_ERR_UNSUPPORTED;
    if ((int64_t)num_blocks * block_size >= ((int64_t)1 << 31)) return PADOC_ERR_INVALID_ARGUMENT;  // int32 slots
    std::vector<uint8_t> seen(num_blocks, 0);
    if (block_order)
        for (int32_t i = 0; i < num_blocks; ++i) {
            const int32_t b = block_order[i];
            if (b < 0 || b >= num_blocks || seen[b]) return PADOC_ERR_INVALID_ARGUMENT;
            seen[b] = 1;
        }
    padoc_mpd *m = new (std::nothrow) padoc_mpd;
    if (!m) return PADOC_ERR_INVALID_ARGUMENT;
    m->bs = block_size;
    m->num_blocks = num_blocks;
    for (int32_t i = 0; i < num_blocks; ++i) m->free_blocks.push_back(block_order ? block_order[i] : i);
    *mpd = m;
    return PADOC_OK;
}

extern "C" void padoc_mpd_destroy(padoc_mpd *mpd) { delete mpd; }

extern "C" padoc_status padoc_mpd_add_page(padoc_mpd *m, int32_t prefix_len, int32_t num_forks, int32_t layout_eos,
                                           int32_t *page_id, int32_t *prefix_slots, int32_t *new_streams)
{
    if (!m || m->in_step || prefix_len < 0 || num_forks < 0 || !page_id || !new_streams) return PADOC_ERR_INVALID_ARGUMENT;
    if (prefix_len > 0 && !prefix_slots) return PADOC_ERR_INVALID_ARGUMENT;
    if (prefix_len >= (1 << 30) || num_forks >= (1 << 30)) return PADOC_ERR_INVALID_ARGUMENT;
    const int32_t need = (prefix_len + m->bs - 1) / m->bs;
    if ((size_t)need > m->free_blocks.size()) return PADOC_ERR_CAPACITY;
    const int32_t pid = (int32_t)m->pages.size();
    m->pages.emplace_back();
    MpdPage &pg = m->pages.back();
    pg.shared_len = prefix_len;
    pg.layout_stream = -1;
    for (int32_t i = 0; i < need; ++i) pg.blocks.push_back(take_block(m));
    for (int32_t t = 0; t < prefix_len; ++t) prefix_slots[t] = pg.blocks[t / m->bs] * m->bs + t % m->bs;
    // the prefill's output: the layout stream lives on unless it is EOS; forks see X only
    if (!layout_eos) pg.layout_stream = new_stream(m, pid, true, 0);
    new_streams[0] = pg.layout_stream;
    for (int32_t f = 0; f < num_forks; ++f) {
        const int32_t id = new_stream(m, pid, false, prefix_len);
        m->pages[pid].branches.push_back(id);
        new_streams[1 + f] = id;
    }
    MpdPage &p2 = m->pages[pid];
    if (page_streams(p2) > 0)
        m->live_pages.push_back(pid);
    else
        give_blocks(m, p2.blocks);   // nothing will ever read the prefix
    *page_id = pid;
    return PADOC_OK;
}

extern "C" padoc_status padoc_mpd_begin_step(padoc_mpd *m, int32_t *num_streams, int32_t *stream_ids,
                                             int32_t *append_slots, int32_t capacity)
{
    if (!m || m->in_step || !num_streams || capacity < 0) return PADOC_ERR_INVALID_ARGUMENT;
    int64_t C = 0, need = 0;
    for (int32_t pid : m->live_pages) {
        const MpdPage &pg = m->pages[pid];
        C += page_streams(pg);
        for (int32_t id : pg.branches) need += m->streams[id].priv_len % m->bs == 0;
        if (pg.layout_stream >= 0) need += pg.shared_len % m->bs == 0;
    }
    if (C > 0 && (!stream_ids || !append_slots)) return PADOC_ERR_INVALID_ARGUMENT;
    if (C > capacity || need > (int64_t)m->free_blocks.size()) return PADOC_ERR_CAPACITY;
    for (int32_t pid : m->live_pages) {
        MpdPage &pg = m->pages[pid];
        if (pg.shared_len >= (1 << 30) - 1) return PADOC_ERR_INVALID_ARGUMENT;
        for (int32_t id : pg.branches)
            if (m->streams[id].priv_len >= (1 << 30) - 1) return PADOC_ERR_INVALID_ARGUMENT;
    }
    m->step_streams.clear();
    int32_t i = 0;
    for (int32_t pid : m->live_pages) {
        MpdPage &pg = m->pages[pid];
        for (int32_t id : pg.branches) {
            MpdStream &s = m->streams[id];
            if (s.priv_len % m->bs == 0) s.blocks.push_back(take_block(m));
            append_slots[i] = s.blocks[s.priv_len / m->bs] * m->bs + s.priv_len % m->bs;
            stream_ids[i++] = id;
            s.priv_len += 1;
            m->step_streams.push_back(id);
        }
        if (pg.layout_stream >= 0) {
            if (pg.shared_len % m->bs == 0) pg.blocks.push_back(take_block(m));
            append_slots[i] = pg.blocks[pg.shared_len / m->bs] * m->bs + pg.shared_len % m->bs;
            stream_ids[i++] = pg.layout_stream;
            pg.shared_len += 1;
            m->step_streams.push_back(pg.layout_stream);
        }
    }
    *num_streams = i;
    m->in_step = true;
    return PADOC_OK;
}

extern "C" padoc_status padoc_mpd_step_shape(const padoc_mpd *m, int32_t *num_pages, int32_t *num_streams,
                                             int32_t *max_page_blocks, int32_t *max_stream_blocks)
{
    if (!m || !m->in_step || !num_pages || !num_streams || !max_page_blocks || !max_stream_blocks)
        return PADOC_ERR_INVALID_ARGUMENT;
    int32_t mp = 0, ms = 0;
    for (int32_t pid : m->live_pages) mp = std::max<int32_t>(mp, (int32_t)m->pages[pid].blocks.size());
    for (int32_t id : m->step_streams) ms = std::max<int32_t>(ms, (int32_t)m->streams[id].blocks.size());
    *num_pages = (int32_t)m->live_pages.size();
    *num_streams = (int32_t)m->step_streams.size();
    *max_page_blocks = mp;
    *max_stream_blocks = ms;
    return PADOC_OK;
}

extern "C" padoc_status padoc_mpd_step_tables(const padoc_mpd *m, int32_t *page_len, padoc_stream_desc *streams,
                                              int32_t *page_table, int32_t page_stride, int32_t *stream_table,
                                              int32_t stream_stride)
{
    if (!m || !m->in_step) return PADOC_ERR_INVALID_ARGUMENT;
    const size_t P = m->live_pages.size(), S = m->step_streams.size();
    int32_t mp = 0, ms = 0;
    for (int32_t pid : m->live_pages) mp = std::max<int32_t>(mp, (int32_t)m->pages[pid].blocks.size());
    for (int32_t id : m->step_streams) ms = std::max<int32_t>(ms, (int32_t)m->streams[id].blocks.size());
    if (page_stride < mp || stream_stride < std::max(ms, 1)) return PADOC_ERR_INVALID_ARGUMENT;
    if (P > 0 && (!page_len || !page_table)) return PADOC_ERR_INVALID_ARGUMENT;
    if (S > 0 && (!streams || !stream_table)) return PADOC_ERR_INVALID_ARGUMENT;
    size_t si = 0;
    for (size_t pi = 0; pi < P; ++pi) {
        const MpdPage &pg = m->pages[m->live_pages[pi]];
        page_len[pi] = pg.shared_len;
        int32_t *row = page_table + pi * (size_t)page_stride;
        std::copy(pg.blocks.begin(), pg.blocks.end(), row);
        std::fill(row + pg.blocks.size(), row + page_stride, -1);
        for (int32_t id : pg.branches) {
            const MpdStream &s = m->streams[id];
            streams[si] = {(int32_t)pi, s.cutoff, s.priv_len};
            int32_t *srow = stream_table + si * (size_t)stream_stride;
            std::copy(s.blocks.begin(), s.blocks.end(), srow);
            std::fill(srow + s.blocks.size(), srow + stream_stride, -1);
            ++si;
        }
        if (pg.layout_stream >= 0) {
            streams[si] = {(int32_t)pi, pg.shared_len, 0};
            std::fill(stream_table + si * (size_t)stream_stride, stream_table + (si + 1) * (size_t)stream_stride, -1);
            ++si;
        }
    }
    return PADOC_OK;
}

extern "C" padoc_status padoc_mpd_end_step(padoc_mpd *m, const int32_t *num_forks, const uint8_t *eos,
                                           int32_t num_streams, int32_t *new_streams, int32_t capacity,
                                           int32_t *num_new)
{
    if (!m || !m->in_step || !num_new || capacity < 0) return PADOC_ERR_INVALID_ARGUMENT;
    if ((size_t)num_streams != m->step_streams.size()) return PADOC_ERR_INVALID_ARGUMENT;
    int64_t total = 0;
    for (int32_t i = 0; i < num_streams; ++i) {
        const int32_t f = num_forks ? num_forks[i] : 0;
        if (f < 0 || f >= (1 << 30)) return PADOC_ERR_INVALID_ARGUMENT;
        if (f > 0 && !m->streams[m->step_streams[i]].layout) return PADOC_ERR_INVALID_ARGUMENT;  // only the layout stream forks
        total += f;
    }
    if (total > 0 && !new_streams) return PADOC_ERR_INVALID_ARGUMENT;
    if (total > capacity) return PADOC_ERR_CAPACITY;
    int32_t k = 0;
    for (int32_t i = 0; i < num_streams; ++i) {
        const int32_t id = m->step_streams[i];
        const int32_t pid = m->streams[id].page;
        const int32_t f = num_forks ? num_forks[i] : 0;
        for (int32_t j = 0; j < f; ++j) {   // copy of the pre-boundary layout row
            const int32_t nid = new_stream(m, pid, false, m->pages[pid].shared_len);
            m->pages[pid].branches.push_back(nid);
            new_streams[k++] = nid;
        }
        if (eos && eos[i]) {
            MpdStream &s = m->streams[id];
            MpdPage &pg = m->pages[pid];
            s.live = false;
            if (s.layout) {
                pg.layout_stream = -1;
            } else {
                give_blocks(m, s.blocks);
                pg.branches.erase(std::find(pg.branches.begin(), pg.branches.end(), id));
            }
        }
    }
    size_t w = 0;
    for (size_t r = 0; r < m->live_pages.size(); ++r) {
        MpdPage &pg = m->pages[m->live_pages[r]];
        if (page_streams(pg) > 0)
            m->live_pages[w++] = m->live_pages[r];
        else
            give_blocks(m, pg.blocks);
    }
    m->live_pages.resize(w);
    m->step_streams.clear();
    m->in_step = false;
    *num_new = k;
    return PADOC_OK;
}

extern "C" padoc_status padoc_mpd_status(const padoc_mpd *m, int32_t *live_pages, int32_t *live_streams,
                                         int32_t *free_blocks)
{
    if (!m || !live_pages || !live_streams || !free_blocks) return PADOC_ERR_INVALID_ARGUMENT;
    int32_t s = 0;
    for (int32_t pid : m->live_pages) s += page_streams(m->pages[pid]);
    *live_pages = (int32_t)m->live_pages.size();
    *live_streams = s;
    *free_blocks = (int32_t)m->free_blocks.size();
    return PADOC_OK;
}

namespace {
int64_t align32(int64_t x) { return (x + 31) & ~(int64_t)31; }
}  // namespace

extern "C" padoc_status padoc_mpd_prepare_step(padoc_mpd *m, const padoc_decode_config *cfg, int32_t *stage,
                                               int64_t capacity_words, padoc_mpd_step *step)
{
    if (!m || !cfg || !step || m->in_step || capacity_words < 0) return PADOC_ERR_INVALID_ARGUMENT;
    if (cfg->block_size != m->bs) return PADOC_ERR_INVALID_ARGUMENT;
    std::memset(step, 0, sizeof(*step));
    // the step's streams and lengths once every live stream has appended its input; nothing changes yet
    std::vector<int32_t> &plen = m->scratch_len;
    std::vector<padoc_stream_desc> &descs = m->scratch_streams;
    plen.clear();
    descs.clear();
    int64_t need = 0;
    int32_t mp = 0, ms = 0;
    for (size_t pi = 0; pi < m->live_pages.size(); ++pi) {
        const MpdPage &pg = m->pages[m->live_pages[pi]];
        if (pg.shared_len >= (1 << 30) - 1) return PADOC_ERR_INVALID_ARGUMENT;
        const int32_t sl = pg.shared_len + (pg.layout_stream >= 0 ? 1 : 0);
        plen.push_back(sl);
        mp = std::max(mp, (sl + m->bs - 1) / m->bs);
        for (int32_t id : pg.branches) {
            const MpdStream &s = m->streams[id];
            if (s.priv_len >= (1 << 30) - 1) return PADOC_ERR_INVALID_ARGUMENT;
            need += s.priv_len % m->bs == 0;
            descs.push_back({(int32_t)pi, s.cutoff, s.priv_len + 1});
            ms = std::max(ms, (s.priv_len + 1 + m->bs - 1) / m->bs);
        }
        if (pg.layout_stream >= 0) {
            need += pg.shared_len % m->bs == 0;
            descs.push_back({(int32_t)pi, sl, 0});
        }
    }
    if (need > (int64_t)m->free_blocks.size()) return PADOC_ERR_CAPACITY;
    const int32_t P = (int32_t)plen.size(), C = (int32_t)descs.size();
    PlanParts &pp = m->plan_parts;
    padoc_status st = padoc_plan_parts_of_list(plen.data(), P, descs.data(), C, cfg, pp);
    if (st != PADOC_OK) return st;
    const int64_t plan_ints = padoc_plan_blob_ints(pp, P, cfg->num_kv_heads);
    const int32_t pstride = std::max(mp, 1), sstride = std::max(ms, 1);
    step->off_plan = 0;
    step->off_page_table = align32(plan_ints);
    step->off_stream_table = step->off_page_table + align32((int64_t)P * pstride);
    step->off_slots = step->off_stream_table + align32((int64_t)C * sstride);
    step->off_rows = step->off_slots + align32(C);
    step->off_first_blocks = step->off_rows + align32(C);
    step->off_stream_ids = step->off_first_blocks + align32((int64_t)pp.num_warps * 4);
    step->upload_words = step->off_stream_ids;
    step->total_words = step->off_stream_ids + align32(C);
    if (capacity_words < step->total_words || !stage) return PADOC_ERR_CAPACITY;
    int32_t n = 0;
    st = padoc_mpd_begin_step(m, &n, stage + step->off_stream_ids, stage + step->off_slots, C);
    if (st != PADOC_OK) return st;
    st = padoc_mpd_step_tables(m, plen.data(), descs.data(), stage + step->off_page_table, pstride,
                               stage + step->off_stream_table, sstride);
    if (st == PADOC_OK) st = padoc_plan_write_blob(pp, P, cfg, stage + step->off_plan, plan_ints, &step->plan);
    if (st != PADOC_OK) return st;   // not reached: both were checked above
    // the pool rows of the first four blocks of each warp's first item, from the tables just
    // written, so that the decode's warps start them before they read their item headers; the block
    // that holds the item's stream's newest row (which the step's append writes) as -2 - row
    int32_t *fb = stage + step->off_first_blocks;
    for (int32_t w = 0; w < pp.num_warps; ++w) {
        int32_t *f = fb + (size_t)w * 4;
        f[0] = f[1] = f[2] = f[3] = -1;
        const int32_t u = pp.num_tc_items + pp.warp_ptr[(size_t)w];
        if (pp.warp_ptr[(size_t)w] >= pp.warp_ptr[(size_t)w + 1]) continue;
        const padoc_item &it = pp.items[(size_t)u];
        const bool shared = it.kind == PADOC_ITEM_SHARED;
        const int32_t *row = shared ? stage + step->off_page_table + (size_t)it.index * pstride
                                    : stage + step->off_stream_table + (size_t)it.first_stream * sstride;
        const int32_t width = shared ? pstride : sstride;
        const int32_t len = shared ? pp.page_len[(size_t)it.index] : pp.streams[(size_t)it.first_stream].private_len;
        const int32_t hot = (len - 1) / m->bs;
        const int32_t b0 = it.tok_begin / m->bs, nb = it.tok_end > it.tok_begin ? (it.tok_end - it.tok_begin + m->bs - 1) / m->bs : 0;
        for (int32_t k = 0; k < 4 && k < nb && b0 + k < width; ++k) {
            const int32_t id = row[b0 + k];
            const int64_t r = ((int64_t)id * cfg->num_kv_heads + it.kv_head) * m->bs;
            if (id < 0 || id >= m->num_blocks || r > INT32_MAX - 2) break;   // left to the decode's own checks
            f[k] = b0 + k == hot ? (int32_t)(-2 - r) : (int32_t)r;
        }
    }
    step->num_streams = n;
    step->num_pages = P;
    step->page_stride = pstride;
    step->stream_stride = sstride;
    return PADOC_OK;
}

extern "C" padoc_status padoc_mpd_launch_step(const padoc_mpd_step *step, const int32_t *stage, int32_t *dev_ints,
                                              int64_t dev_capacity_words, const padoc_kv_pool *pool,
                                              const void *k_src, const void *v_src, const void *q_src,
                                              int64_t src_total, void *q_dst, float scale, void *out, float *lse,
                                              void *workspace, size_t workspace_bytes, padoc_stream_t stream)
{
    if (!step || !dev_ints || !pool) return PADOC_ERR_INVALID_ARGUMENT;
    const int32_t C = step->num_streams;
    if (C == 0) return PADOC_OK;
    if (C < 0 || step->upload_words < 0 || dev_capacity_words < step->upload_words || (((uintptr_t)dev_ints) & 255))
        return PADOC_ERR_INVALID_ARGUMENT;
    const padoc_decode_plan &info = step->plan;
    if (info.num_streams != C || step->off_plan + info.plan_ints > step->upload_words ||
        step->off_rows + C > step->upload_words)
        return PADOC_ERR_INVALID_ARGUMENT;
    if (stage && cudaMemcpyAsync(dev_ints, stage, (size_t)step->upload_words * sizeof(int32_t), cudaMemcpyHostToDevice,
                                 (cudaStream_t)stream) != cudaSuccess)
        return PADOC_ERR_CUDA;
    padoc_status st = padoc_append_inputs(pool, k_src, v_src, q_src, src_total, info.cfg.num_q_heads, q_dst,
                                          dev_ints + step->off_rows, dev_ints + step->off_slots, C, stream);
    if (st != PADOC_OK) return st;
    return padoc_branch_decode_attn_after_append(pool, &info, dev_ints + step->off_plan, dev_ints + step->off_page_table,
                                    step->page_stride, dev_ints + step->off_stream_table, step->stream_stride, q_dst,
                                    scale, out, lse, workspace, workspace_bytes, stream,
                                                 step->plan.num_warps > 0 ? dev_ints + step->off_first_blocks : nullptr);
}

// ---- the step loop's host side in one call per step (padoc_mpd_runner_*) ----------------------

struct padoc_mpd_runner {
    padoc_mpd *m = nullptr;
    padoc_decode_config cfg{};
    padoc_kv_pool pool{};
    int32_t *stage[2] = {nullptr, nullptr};   // pinned host staging, used in turn
    int64_t stage_words[2] = {0, 0};
    cudaEvent_t copied[2] = {nullptr, nullptr};   // recorded after the step whose stage it is
    bool recorded[2] = {false, false};
    int32_t *dev_ints = nullptr;
    int64_t dev_words = 0;
    void *q_step = nullptr;
    size_t q_bytes = 0;
    void *workspace = nullptr;
    size_t workspace_bytes = 0;
    int64_t turn = 0;
    int last = -1;                 // stage of the last prepared step
    padoc_mpd_step last_step{};
};

namespace {

void runner_free(padoc_mpd_runner *r)
{
    for (int b = 0; b < 2; ++b) {
        if (r->copied[b]) {
            if (r->recorded[b]) cudaEventSynchronize(r->copied[b]);
            cudaEventDestroy(r->copied[b]);
        }
        if (r->stage[b]) cudaFreeHost(r->stage[b]);
    }
    cudaFree(r->dev_ints);   // the events above cover every launch that read these
    cudaFree(r->q_step);
    cudaFree(r->workspace);
}

// Grows a device buffer to at least `need` bytes (twice the old size at least). The stream is
// drained first: the step in flight may still read the old buffer.
padoc_status grow_device(void **buf, size_t *bytes, size_t need, cudaStream_t stream)
{
    if (need <= *bytes) return PADOC_OK;
    const size_t nb = std::max(need, 2 * *bytes);
    if (*buf) {
        if (cudaStreamSynchronize(stream) != cudaSuccess) return PADOC_ERR_CUDA;
        cudaFree(*buf);
        *buf = nullptr;
        *bytes = 0;
    }
    if (cudaMalloc(buf, nb) != cudaSuccess) {
        *buf = nullptr;
        return PADOC_ERR_CUDA;
    }
    *bytes = nb;
    return PADOC_OK;
}

}  // namespace

extern "C" padoc_status padoc_mpd_runner_create(padoc_mpd *m, const padoc_decode_config *cfg,
                                                const padoc_kv_pool *pool, padoc_mpd_runner **runner)
{
    if (!m || !cfg || !pool || !runner) return PADOC_ERR_INVALID_ARGUMENT;
    if (cfg->block_size != m->bs || pool->block_size != m->bs || pool->num_blocks < m->num_blocks ||
        pool->num_kv_heads != cfg->num_kv_heads || pool->head_dim != cfg->head_dim || cfg->layout_streams)
        return PADOC_ERR_INVALID_ARGUMENT;
    padoc_mpd_runner *r = new (std::nothrow) padoc_mpd_runner;
    if (!r) return PADOC_ERR_INVALID_ARGUMENT;
    r->m = m;
    r->cfg = *cfg;
    r->pool = *pool;
    for (int b = 0; b < 2; ++b)
        if (cudaEventCreateWithFlags(&r->copied[b], cudaEventDisableTiming) != cudaSuccess) {
            r->copied[b] = nullptr;
            runner_free(r);
            delete r;
            return PADOC_ERR_CUDA;
        }
    *runner = r;
    return PADOC_OK;
}

extern "C" void padoc_mpd_runner_destroy(padoc_mpd_runner *r)
{
    if (!r) return;
    runner_free(r);
    delete r;
}

extern "C" padoc_status padoc_mpd_runner_step(padoc_mpd_runner *r, const padoc_mpd_run_args *a, int32_t *num_streams,
                                              int64_t *upload_bytes)
{
    if (!r || !a || !num_streams) return PADOC_ERR_INVALID_ARGUMENT;
    if (upload_bytes) *upload_bytes = 0;
    padoc_mpd *m = r->m;
    if (m->in_step || a->src_total < 0 || a->out_rows < 0 || a->ids_capacity < 0) return PADOC_ERR_INVALID_ARGUMENT;
    // what the step needs of the caller's arrays, checked before anything begins
    int64_t C = 0;
    for (int32_t pid : m->live_pages) C += page_streams(m->pages[pid]);
    if (C > a->out_rows || C > a->ids_capacity) return PADOC_ERR_CAPACITY;
    if (C > 0 && (!a->stream_ids || !a->src_row_of_stream || !a->k_src || !a->v_src || !a->q_src || !a->out ||
                  !a->lse))
        return PADOC_ERR_INVALID_ARGUMENT;
    if (C > 0 && (int64_t)a->num_stream_ids < (int64_t)m->streams.size()) return PADOC_ERR_INVALID_ARGUMENT;
    const cudaStream_t stream = (cudaStream_t)a->stream;
    const int b = (int)(r->turn & 1);
    if (r->recorded[b]) {   // the copy that read this stage two steps ago (usually done: ask first)
        const cudaError_t q = cudaEventQuery(r->copied[b]);
        if (q != cudaSuccess && (q != cudaErrorNotReady || cudaEventSynchronize(r->copied[b]) != cudaSuccess))
            return PADOC_ERR_CUDA;
        r->recorded[b] = false;
    }
    padoc_mpd_step step;
    padoc_status st;
    for (;;) {
        st = padoc_mpd_prepare_step(m, &r->cfg, r->stage[b], r->stage_words[b], &step);
        if (st != PADOC_ERR_CAPACITY || step.total_words <= r->stage_words[b]) break;
        // a larger stage (nothing has begun): no copy reads this one any more
        if (r->stage[b]) cudaFreeHost(r->stage[b]);
        r->stage[b] = nullptr;
        r->stage_words[b] = 0;
        const int64_t words = std::max<int64_t>(step.total_words * 2, 1 << 16);
        void *p = nullptr;
        if (cudaHostAlloc(&p, (size_t)words * sizeof(int32_t), cudaHostAllocDefault) != cudaSuccess)
            return PADOC_ERR_CUDA;
        r->stage[b] = static_cast<int32_t *>(p);
        r->stage_words[b] = words;
    }
    if (st != PADOC_OK) return st;
    ++r->turn;
    r->last = b;
    r->last_step = step;
    const int32_t n = step.num_streams;
    *num_streams = n;
    if (n == 0) return PADOC_OK;
    int32_t *stage = r->stage[b];
    const int32_t *ids = stage + step.off_stream_ids;
    std::memcpy(a->stream_ids, ids, (size_t)n * sizeof(int32_t));
    for (int32_t i = 0; i < n; ++i) stage[step.off_rows + i] = a->src_row_of_stream[ids[i]];
    // device buffers for this step (the stream is drained before one is replaced)
    const size_t elt = r->pool.dtype == PADOC_DTYPE_BF16 ? 2 : 4;
    size_t ws = 0, dev_bytes = (size_t)r->dev_words * sizeof(int32_t);
    padoc_decode_workspace_size(&step.plan, &ws);
    st = grow_device(reinterpret_cast<void **>(&r->dev_ints), &dev_bytes, (size_t)step.upload_words * sizeof(int32_t),
                     stream);
    r->dev_words = (int64_t)(dev_bytes / sizeof(int32_t));
    if (st == PADOC_OK)
        st = grow_device(&r->q_step, &r->q_bytes, (size_t)n * r->cfg.num_q_heads * r->cfg.head_dim * elt, stream);
    if (st == PADOC_OK) st = grow_device(&r->workspace, &r->workspace_bytes, std::max<size_t>(ws, 256), stream);
    if (st != PADOC_OK) return st;
    st = padoc_mpd_launch_step(&step, stage, r->dev_ints, r->dev_words, &r->pool, a->k_src, a->v_src, a->q_src,
                               a->src_total, r->q_step, a->scale, a->out, a->lse, r->workspace, r->workspace_bytes,
                               a->stream);
    if (st != PADOC_OK) return st;
    if (cudaEventRecord(r->copied[b], stream) != cudaSuccess) return PADOC_ERR_CUDA;
    r->recorded[b] = true;
    if (upload_bytes) *upload_bytes = step.upload_words * (int64_t)sizeof(int32_t);
    return PADOC_OK;
}

extern "C" padoc_status padoc_mpd_runner_last_step(const padoc_mpd_runner *r, padoc_mpd_step *step,
                                                   const int32_t **stage)
{
    if (!r || !step || !stage || r->last < 0) return PADOC_ERR_INVALID_ARGUMENT;
    *step = r->last_step;
    *stage = r->stage[r->last];
    return PADOC_OK;
}
