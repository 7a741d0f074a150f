// decode.cu -- C2/C4/C5: one decode step for every live stream over the paged KV cache
// (Algorithm 1's "decode o for all streams using the additive bias A_M", App. E.1), the split-K
// merge of partial softmax results, and the fp32 bring-up path.
//
// bf16 path. The planner cuts each page's shared stream into split-K pieces and each stream's
// private rows into pieces; a work item is one piece for one KV head. Pages whose branches x
// query heads fill dense M = 128 tiles read their shared stream on the tensor cores
// (decode_tc.cu): each K/V tile is fetched once for all of the page's streams. Every private
// history, and the shared stream of pages with few branches, is read by the warp path
// (decode_warp.cuh), which the same grid runs (bf16): its CTAs run their tensor-core pieces first,
// the rest start on the warp lists at once; for the E4M3 pool the warp lists run in a grid of their
// own. A split-K merge then joins each (stream, head)'s partials.
#include <math.h>
#include <stddef.h>

#include <mutex>

#include "common.cuh"
#include "decode_warp.cuh"
#include "plan_build.h"

namespace {

using namespace padoc_warp;

constexpr size_t kDecodeSmemE4M3 = 1024 + kRingBytesE4M3;   // + the slack to align the base by hand

// The warp lists as a grid of their own (the E4M3 pool), 8 warps per CTA, launched as a programmatic
// dependent of the tensor-core grid when there is one. Warp CTA c is CTA c: the first ones take the
// SMs the tensor-core grid leaves free, the others start as its CTAs end.
template <bool kE4M3>
__global__ void __launch_bounds__(kWarps * 32, 1)
decode_warp_kernel(const DecodeParams prm, int after_tc)
{
    // the merge that follows waits for this whole grid before it reads anything, so it may launch now
    pdl_launch_dependents();
    // Without a tensor-core grid this grid is a programmatic dependent of whatever kernel precedes
    // it in the stream (the previous step's merge, which may still read partials, or the kernel
    // that wrote the queries and the new K/V rows): it waits for that kernel before any global
    // access, so only its launch overlaps the previous kernel. After a tensor-core grid (which waited
    // for that kernel already) each warp waits for it before it ends, so that the merge sees both
    // grids' partials.
    if (!after_tc) pdl_wait_prerequisite();
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int wi = blockIdx.x * kWarps + warp;
    if (wi < prm.num_warps) decode_warp_role<kE4M3>(prm, smem, warp, lane, wi);
    if (after_tc) pdl_wait_prerequisite();
}

// ------------------------------------------------------------------------------------------------
// Split-K merge (C4): one warp per output row, 4 consecutive dims per lane.
// ------------------------------------------------------------------------------------------------
struct UniformSlots {  // public combine: part_row = split * rows + row
    int32_t splits;
    int64_t rows;
    __device__ int count(int64_t) const { return splits; }
    __device__ int64_t part_row(int64_t row, int i) const { return (int64_t)i * rows + row; }
};

// Decode merge: one CTA per (stream, KV head), 16 dim chunks x its 8 query heads, each thread 8 of
// the 128 dims of one head. One pass over the slots with an online reference (the running max of lse_s): four
// partials' LSE and O loads are in flight per thread at a time. Registers are capped so that nine CTAs
// fit on an SM: the serving batch's 1344 (stream, KV head) pairs then start in one wave.

// The online pass of one thread over the key's slots in blocks of four, blocks b0, b0 + stride, ...:
// (mref, ssum, acc) hold the running reference, the weights' sum and the weighted O sums.
struct MergeState {
    float mref = -INFINITY, ssum = 0.f;
    float4 acc0 = make_float4(0.f, 0.f, 0.f, 0.f), acc1 = make_float4(0.f, 0.f, 0.f, 0.f);
};
// bo: this thread's 8 dims of its head in the key's first slot (bf16 partials, a slot every
// kGroup * kD values); bl: its head's LSE in the first slot. kPer partials' loads in flight.
template <int kPer>
__device__ __forceinline__ void merge_slots(const __nv_bfloat16 *bo, const float *bl, int n, int b0, int stride,
                                            MergeState &ms)
{
    constexpr size_t kSlotO = (size_t)kGroup * kD;
    for (int i = kPer * b0; i < n; i += kPer * stride) {
        float li[kPer];
        uint4 v[kPer];
#pragma unroll
        for (int u = 0; u < kPer; ++u) {
            const bool in = i + u < n;
            li[u] = in ? bl[(size_t)(i + u) * kGroup] : -INFINITY;
            v[u] = in ? *reinterpret_cast<const uint4 *>(bo + (i + u) * kSlotO) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < kPer; ++u) {
            if (li[u] == -INFINITY) continue;   // an empty partial weighs nothing
            if (li[u] > ms.mref) {
                const float a = ms.mref == -INFINITY ? 0.f : expf(ms.mref - li[u]);
                ms.ssum *= a;
                ms.acc0.x *= a; ms.acc0.y *= a; ms.acc0.z *= a; ms.acc0.w *= a;
                ms.acc1.x *= a; ms.acc1.y *= a; ms.acc1.z *= a; ms.acc1.w *= a;
                ms.mref = li[u];
            }
            const float w = expf(li[u] - ms.mref);
            ms.ssum += w;
            // bf16 to fp32: the upper 16 bits of each float
            ms.acc0.x += w * __uint_as_float(v[u].x << 16); ms.acc0.y += w * __uint_as_float(v[u].x & 0xffff0000u);
            ms.acc0.z += w * __uint_as_float(v[u].y << 16); ms.acc0.w += w * __uint_as_float(v[u].y & 0xffff0000u);
            ms.acc1.x += w * __uint_as_float(v[u].z << 16); ms.acc1.y += w * __uint_as_float(v[u].z & 0xffff0000u);
            ms.acc1.z += w * __uint_as_float(v[u].w << 16); ms.acc1.w += w * __uint_as_float(v[u].w & 0xffff0000u);
        }
    }
}

// Joins state o into ms (both over disjoint sets of partials, each with its own reference).
__device__ __forceinline__ void merge_join(MergeState &ms, const MergeState &o)
{
    if (o.mref == -INFINITY) return;   // that state saw no partial with weight
    const float m = fmaxf(ms.mref, o.mref);
    const float a = ms.mref == -INFINITY ? 0.f : expf(ms.mref - m), b = expf(o.mref - m);
    ms.ssum = ms.ssum * a + o.ssum * b;
    ms.acc0.x = ms.acc0.x * a + o.acc0.x * b; ms.acc0.y = ms.acc0.y * a + o.acc0.y * b;
    ms.acc0.z = ms.acc0.z * a + o.acc0.z * b; ms.acc0.w = ms.acc0.w * a + o.acc0.w * b;
    ms.acc1.x = ms.acc1.x * a + o.acc1.x * b; ms.acc1.y = ms.acc1.y * a + o.acc1.y * b;
    ms.acc1.z = ms.acc1.z * a + o.acc1.z * b; ms.acc1.w = ms.acc1.w * a + o.acc1.w * b;
    ms.mref = m;
}

__device__ __forceinline__ void merge_store(const MergeState &ms, int key, int h, int part, __nv_bfloat16 *out,
                                            float *lse_out)
{
    const float inv = ms.ssum > 0.f ? 1.f / ms.ssum : 0.f;
    uint4 pk;
    pk.x = pack_bf16x2(ms.acc0.x * inv, ms.acc0.y * inv); pk.y = pack_bf16x2(ms.acc0.z * inv, ms.acc0.w * inv);
    pk.z = pack_bf16x2(ms.acc1.x * inv, ms.acc1.y * inv); pk.w = pack_bf16x2(ms.acc1.z * inv, ms.acc1.w * inv);
    *reinterpret_cast<uint4 *>(out + ((size_t)key * kGroup + h) * kD + part * 8) = pk;
    if (part == 0) lse_out[(size_t)key * kGroup + h] = ms.ssum > 0.f ? ms.mref + logf(ms.ssum) : -INFINITY;
}

// kIndexed: CTA b joins key merge_keys[b] (a plan whose sole items write some keys directly);
// otherwise every key is merged and CTA b joins key b (no index kept live: nine CTAs per SM need the
// 56-register cap).
template <bool kIndexed>
__global__ void __launch_bounds__(128, 9) decode_combine_kernel(const int32_t *__restrict__ slot_ptr,
                                                             const int32_t *__restrict__ merge_keys,
                                                             const __nv_bfloat16 *__restrict__ part_o,
                                                             const float *__restrict__ part_lse,
                                                             __nv_bfloat16 *__restrict__ out, float *__restrict__ lse_out)
{
    // The slot range comes from the plan, which no kernel of the step writes, so it is read before
    // the wait. Launched programmatically after the decode grid: wait for it (and its partials),
    // then let the next step's first kernel launch (it waits for this grid before touching memory).
    const int key = kIndexed ? merge_keys[blockIdx.x] : (int)blockIdx.x;   // s * Hkv + g; output rows key * 8 + h
    const int p0 = slot_ptr[key], n = slot_ptr[key + 1] - p0;
    pdl_wait_prerequisite();
    pdl_launch_dependents();
    const int tid = threadIdx.x;
    const int h = tid & 7, part = tid >> 3;          // head, 8-dim chunk: a warp reads 4 chunks x 8 heads, contiguous
    const __nv_bfloat16 *bo = part_o + (size_t)p0 * kGroup * kD + (part * kGroup + h) * 8;   // chunk `part` of head h
    const float *bl = part_lse + (size_t)p0 * kGroup + h;
    MergeState ms;
    merge_slots<6>(bo, bl, n, 0, 1, ms);
    merge_store(ms, key, h, part, out, lse_out);
}

// The merge for steps with few keys and many partials each (a decoding loop's small steps): kGroups
// groups of 128 threads share a key, group q taking the blocks of four slots q, q + kGroups, ...,
// and group 0 joins the running states through shared memory. Launched instead of
// decode_combine_kernel for keys of more than 8 partials when the keys fit in one wave of these CTAs
// (two per SM) and the cluster merge below is not taken.
template <bool kIndexed, int kGroups>
__global__ void __launch_bounds__(128 * kGroups, 8 / kGroups) decode_combine_wide_kernel(
    const int32_t *__restrict__ slot_ptr, const int32_t *__restrict__ merge_keys, const __nv_bfloat16 *__restrict__ part_o,
    const float *__restrict__ part_lse, __nv_bfloat16 *__restrict__ out, float *__restrict__ lse_out)
{
    constexpr int kWideGroups = kGroups;
    const int key = kIndexed ? merge_keys[blockIdx.x] : (int)blockIdx.x;
    const int p0 = slot_ptr[key], n = slot_ptr[key + 1] - p0;
    pdl_wait_prerequisite();
    pdl_launch_dependents();
    const int tid = threadIdx.x & 127, q = threadIdx.x >> 7;
    const int h = tid & 7, part = tid >> 3;
    const __nv_bfloat16 *bo = part_o + (size_t)p0 * kGroup * kD + (part * kGroup + h) * 8;
    const float *bl = part_lse + (size_t)p0 * kGroup + h;
    MergeState ms;
    merge_slots<4>(bo, bl, n, q, kWideGroups, ms);
    __shared__ MergeState st[kWideGroups - 1][128];
    if (q > 0) st[q - 1][tid] = ms;
    __syncthreads();
    if (q > 0) return;
#pragma unroll
    for (int k = 0; k < kWideGroups - 1; ++k) merge_join(ms, st[k][tid]);
    merge_store(ms, key, h, part, out, lse_out);
}

// The merge for keys with very many partials (a decoding loop's small steps cut into short items):
// one thread-block cluster of kMergeCluster CTAs per key, so that the key's partials are read by as
// many SMs. Group q of CTA r takes the blocks of four slots r + kMergeCluster q, then every
// 4 kMergeCluster-th block; each CTA joins its four groups in shared memory, and CTA 0 joins the
// CTAs' states through distributed shared memory and writes the key's outputs. Two cluster
// barriers: the CTAs' states are complete before CTA 0 reads them, and stay until it has.
constexpr int kMergeCluster = 8;
#ifndef PADOC_MERGE_CLUSTER_MAX_KEYS
#define PADOC_MERGE_CLUSTER_MAX_KEYS 8
#endif

__device__ __forceinline__ uint32_t cluster_ctarank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ void cluster_barrier()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// The state at shared address `addr` of cluster CTA `rank`.
__device__ __forceinline__ MergeState load_remote_state(uint32_t addr, uint32_t rank)
{
    uint32_t ra;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(addr), "r"(rank));
    MergeState o;
    asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(o.mref), "=f"(o.ssum) : "r"(ra) : "memory");
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(o.acc0.x), "=f"(o.acc0.y), "=f"(o.acc0.z), "=f"(o.acc0.w)
                 : "r"(ra + (uint32_t)offsetof(MergeState, acc0))
                 : "memory");
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(o.acc1.x), "=f"(o.acc1.y), "=f"(o.acc1.z), "=f"(o.acc1.w)
                 : "r"(ra + (uint32_t)offsetof(MergeState, acc1))
                 : "memory");
    return o;
}

template <bool kIndexed>
__global__ void __launch_bounds__(512, 2) decode_combine_cluster_kernel(
    const int32_t *__restrict__ slot_ptr, const int32_t *__restrict__ merge_keys, const __nv_bfloat16 *__restrict__ part_o,
    const float *__restrict__ part_lse, __nv_bfloat16 *__restrict__ out, float *__restrict__ lse_out)
{
    const uint32_t rank = cluster_ctarank();
    const int kidx = (int)(blockIdx.x / kMergeCluster);
    const int key = kIndexed ? merge_keys[kidx] : kidx;
    const int p0 = slot_ptr[key], n = slot_ptr[key + 1] - p0;
    pdl_wait_prerequisite();
    pdl_launch_dependents();
    const int tid = threadIdx.x & 127, q = threadIdx.x >> 7;
    const int h = tid & 7, part = tid >> 3;
    const __nv_bfloat16 *bo = part_o + (size_t)p0 * kGroup * kD + (part * kGroup + h) * 8;
    const float *bl = part_lse + (size_t)p0 * kGroup + h;
    MergeState ms;
    merge_slots<4>(bo, bl, n, (int)rank + kMergeCluster * q, 4 * kMergeCluster, ms);
    __shared__ MergeState st[4][128];
    st[q][tid] = ms;
    __syncthreads();
    if (q == 0) {
#pragma unroll
        for (int k = 1; k < 4; ++k) merge_join(ms, st[k][tid]);
        st[0][tid] = ms;
    }
    cluster_barrier();
    if (rank == 0 && q == 0) {
        const uint32_t addr = smem_u32(&st[0][tid]);
#pragma unroll 1
        for (uint32_t r = 1; r < (uint32_t)kMergeCluster; ++r) merge_join(ms, load_remote_state(addr, r));
        merge_store(ms, key, h, part, out, lse_out);
    }
    cluster_barrier();
}

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
            int i = 0;
            for (; i + 4 <= n; i += 4) {   // four partials in flight at a time
                float w[4];
                float4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int64_t pr = sl.part_row(row, i + u);
                    w[u] = expf(part_lse[pr] - tot);
                    v[u] = *reinterpret_cast<const float4 *>(part_o + pr * d + c0);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (w[u] != 0.f) { acc.x += w[u] * v[u].x; acc.y += w[u] * v[u].y; acc.z += w[u] * v[u].z; acc.w += w[u] * v[u].w; }
            }
            for (; i < n; ++i) {
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

// The bf16 path's split-K decode over either pool: the tensor-core grid for the shared streams of
// dense pages, the warp grid for the rest, and the merge; arguments validated by the caller.
struct DecodePool {
    bool e4m3;
    const void *k, *v;                    // bf16 pools or E4M3 codes
    const float *k_scales, *v_scales;     // E4M3 scales
    int32_t num_blocks;
};

padoc_status decode_split_k(const DecodePool &pl, const padoc_decode_plan *info, const int32_t *plan,
                            const int32_t *page_block_table, int32_t page_table_stride,
                            const int32_t *stream_block_table, int32_t stream_table_stride, const void *q, float scale,
                            void *out, float *lse, void *workspace, size_t workspace_bytes, cudaStream_t cs,
                            bool after_append = false, const int32_t *first_blocks = nullptr)
{
    const padoc_decode_config &cfg = info->cfg;
    if (cfg.head_dim != kD || cfg.num_q_heads != kGroup * cfg.num_kv_heads || cfg.block_size != kBlk)
        return PADOC_ERR_UNSUPPORTED;
    size_t need = 0;
    const padoc_status ws_st = padoc_decode_workspace_size(info, &need);
    if (ws_st != PADOC_OK) return ws_st;
    if (!workspace || workspace_bytes < need) return PADOC_ERR_WORKSPACE_TOO_SMALL;
    if (((uintptr_t)workspace) & 255) return PADOC_ERR_INVALID_ARGUMENT;
    int *err = padoc_device_error_word();   // the first CUDA call: every check above is on the host
    if (!err) return PADOC_ERR_CUDA;

    const uint64_t rows = (uint64_t)pl.num_blocks * cfg.num_kv_heads * kBlk;
    CUtensorMap kmap, vmap;   // bf16: 16-row x 64-column boxes; E4M3: 16-row x 128-byte boxes of codes
    if (pl.e4m3 ? (!padoc_make_tmap_u8(&kmap, pl.k, kD, rows, kD, kD, kBlk) ||
                   !padoc_make_tmap_u8(&vmap, pl.v, kD, rows, kD, kD, kBlk))
                : (!padoc_make_tmap_bf16(&kmap, pl.k, kD, rows, kD * 2, 64, kBlk) ||
                   !padoc_make_tmap_bf16(&vmap, pl.v, kD, rows, kD * 2, 64, kBlk)))
        return PADOC_ERR_CUDA;

    if ((int64_t)pl.num_blocks * cfg.num_kv_heads * kBlk >= INT32_MAX) return PADOC_ERR_UNSUPPORTED;
    __nv_bfloat16 *part_o = (__nv_bfloat16 *)workspace;
    float *part_lse = (float *)((uint8_t *)workspace + padoc_align256((size_t)info->num_slots * kGroup * kD * 2));
    const float sl2 = scale * PADOC_LOG2E;

    // shared streams of dense pages on the tensor cores
    CUtensorMap qmap = {};   // Q [S][Hq][d] as [S][Hkv][8][d]: a box is 16 streams x the 8 heads of one KV head
    {
        const uint64_t dims[4] = {(uint64_t)kD, (uint64_t)kGroup, (uint64_t)cfg.num_kv_heads, (uint64_t)info->num_streams};
        const uint64_t strides[3] = {(uint64_t)kD * 2, (uint64_t)kGroup * kD * 2, (uint64_t)cfg.num_q_heads * kD * 2};
        const uint32_t box[4] = {64, (uint32_t)kGroup, 1, 16};
        if (info->num_tc_items > 0 && !padoc_make_tmap_bf16_4d(&qmap, q, dims, strides, box)) return PADOC_ERR_CUDA;
    }
    // private histories and the shared streams of sparse pages, one warp per item
    DecodeParams prm;
    prm.stream_page = plan + info->off_stream_page;
    prm.shared_len = plan + info->off_shared_len;
    prm.private_len = plan + info->off_private_len;
    prm.slot_ptr = plan + info->off_slot_ptr;
    prm.page_len = plan + info->off_page_len;
    prm.pre_wait = after_append && !pl.e4m3 ? 1 : 0;
    prm.first_blocks = prm.pre_wait ? first_blocks : nullptr;
    prm.items = reinterpret_cast<const padoc_item *>(plan + info->off_items);
    prm.first_item = info->num_tc_items;
    prm.warp_ptr = plan + info->off_warp_ptr;
    prm.num_warps = info->num_warps;
    prm.page_table = page_block_table;
    prm.stream_table = stream_block_table;
    prm.page_stride = page_table_stride;
    prm.stream_stride = stream_table_stride;
    prm.num_blocks = pl.num_blocks;
    prm.num_kv_heads = cfg.num_kv_heads;
    prm.num_q_heads = cfg.num_q_heads;
    prm.pool_rows = pl.num_blocks * cfg.num_kv_heads * kBlk;
    prm.k_pool = pl.e4m3 ? nullptr : (const __nv_bfloat16 *)pl.k;
    prm.v_pool = pl.e4m3 ? nullptr : (const __nv_bfloat16 *)pl.v;
    prm.k_codes = pl.e4m3 ? (const uint8_t *)pl.k : nullptr;
    prm.v_codes = pl.e4m3 ? (const uint8_t *)pl.v : nullptr;
    prm.k_scales = pl.k_scales;
    prm.v_scales = pl.v_scales;
    prm.q = (const __nv_bfloat16 *)q;
    prm.part_o = part_o;
    prm.part_lse = part_lse;
    prm.scale_log2 = sl2;
    prm.err = err;
    // the decode grid: tensor-core pieces, then (bf16: on those CTAs and on the SMs they leave free)
    // the warp lists
    padoc_status st = padoc_launch_decode_tc(&kmap, &vmap, &qmap, plan, info, page_block_table, page_table_stride,
                                             stream_block_table, stream_table_stride, pl.num_blocks,
                                             pl.e4m3 ? pl.k_scales : nullptr, pl.e4m3 ? pl.v_scales : nullptr,
                                             part_o, part_lse, (__nv_bfloat16 *)out, lse, sl2, err, &prm, cs);
    if (st != PADOC_OK) return st;
    if (pl.e4m3 && prm.num_warps > 0) {   // E4M3: the warp lists in a grid of their own
        const int after_tc = info->num_tc_items > 0 ? 1 : 0;
        st = padoc_set_max_smem(reinterpret_cast<const void *>(decode_warp_kernel<true>), (int)kDecodeSmemE4M3);
        if (st != PADOC_OK) return st;
        cudaLaunchConfig_t lc = {};
        lc.gridDim = dim3((unsigned)((prm.num_warps + kWarps - 1) / kWarps));
        lc.blockDim = dim3(kWarps * 32);
        lc.dynamicSmemBytes = kDecodeSmemE4M3;
        lc.stream = cs;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        lc.attrs = attr;
        lc.numAttrs = 1;
        PADOC_CUDA_TRY(cudaLaunchKernelEx(&lc, decode_warp_kernel<true>, prm, after_tc));
        st = padoc_launch_status();
        if (st != PADOC_OK) return st;
    }
    if (info->num_merge_keys > 0) {   // the keys with more than one partial (or a warp item's one)
        cudaLaunchConfig_t lc = {};
        lc.gridDim = dim3((unsigned)info->num_merge_keys);
        lc.blockDim = dim3(128);
        lc.stream = cs;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // see the kernel's wait
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        lc.attrs = attr;
        lc.numAttrs = 1;
        const bool all_keys = (int64_t)info->num_merge_keys == (int64_t)info->num_streams * cfg.num_kv_heads;
        // few keys with many partials each: four or eight thread groups per key, in one wave
        const int sms = padoc_default_ctas();
        // very many partials per key and few keys: a cluster of CTAs per key
        const bool clustered = info->max_stream_slots > 32 && info->num_merge_keys <= PADOC_MERGE_CLUSTER_MAX_KEYS;
        const bool wide = !clustered && info->max_stream_slots > 8 && info->num_merge_keys <= 2 * sms;
        cudaLaunchAttribute cattr[2];
        if (clustered) {
            lc.gridDim = dim3((unsigned)(info->num_merge_keys * kMergeCluster));
            lc.blockDim = dim3(512);
            cattr[0] = attr[0];
            cattr[1].id = cudaLaunchAttributeClusterDimension;
            cattr[1].val.clusterDim.x = kMergeCluster;
            cattr[1].val.clusterDim.y = 1;
            cattr[1].val.clusterDim.z = 1;
            lc.attrs = cattr;
            lc.numAttrs = 2;
        } else if (wide) {
            lc.blockDim = dim3(512);
        }
        auto kern = clustered ? (all_keys ? decode_combine_cluster_kernel<false> : decode_combine_cluster_kernel<true>)
                    : wide    ? (all_keys ? decode_combine_wide_kernel<false, 4> : decode_combine_wide_kernel<true, 4>)
                              : (all_keys ? decode_combine_kernel<false> : decode_combine_kernel<true>);
        PADOC_CUDA_TRY(cudaLaunchKernelEx(&lc, kern, prm.slot_ptr, (const int32_t *)(plan + info->off_merge_keys),
                                          (const __nv_bfloat16 *)part_o, (const float *)part_lse, (__nv_bfloat16 *)out, lse));
    }
    return padoc_launch_status();
}

}  // namespace

// ------------------------------------------------------------------------------------------------
// Host entry points
// ------------------------------------------------------------------------------------------------

namespace {

padoc_status branch_decode(const padoc_kv_pool *pool, const padoc_decode_plan *info, const int32_t *plan_dev,
                           const int32_t *page_block_table, int32_t page_table_stride,
                           const int32_t *stream_block_table, int32_t stream_table_stride, const void *q, float scale,
                           void *out, float *lse, void *workspace, size_t workspace_bytes, padoc_stream_t stream,
                           bool after_append, const int32_t *first_blocks = nullptr)
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
    cudaStream_t cs = (cudaStream_t)stream;

    if (pool->dtype == PADOC_DTYPE_F32) {
        int *err = padoc_device_error_word();
        if (!err) return PADOC_ERR_CUDA;
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
    const DecodePool dp{false, pool->k_pool, pool->v_pool, nullptr, nullptr, pool->num_blocks};
    return decode_split_k(dp, info, plan, page_block_table, page_table_stride, stream_block_table, stream_table_stride,
                          q, scale, out, lse, workspace, workspace_bytes, cs, after_append, first_blocks);
}

}  // namespace

extern "C" padoc_status padoc_branch_decode_attn(const padoc_kv_pool *pool, const padoc_decode_plan *info,
                                                 const int32_t *plan_dev, const int32_t *page_block_table,
                                                 int32_t page_table_stride, const int32_t *stream_block_table,
                                                 int32_t stream_table_stride, const void *q, float scale, void *out,
                                                 float *lse, void *workspace, size_t workspace_bytes,
                                                 padoc_stream_t stream)
{
    return branch_decode(pool, info, plan_dev, page_block_table, page_table_stride, stream_block_table,
                         stream_table_stride, q, scale, out, lse, workspace, workspace_bytes, stream, false);
}

padoc_status padoc_branch_decode_attn_after_append(const padoc_kv_pool *pool, const padoc_decode_plan *info,
                                                   const int32_t *plan_dev, const int32_t *page_block_table,
                                                   int32_t page_table_stride, const int32_t *stream_block_table,
                                                   int32_t stream_table_stride, const void *q, float scale, void *out,
                                                   float *lse, void *workspace, size_t workspace_bytes,
                                                   padoc_stream_t stream, const int32_t *first_blocks)
{
    return branch_decode(pool, info, plan_dev, page_block_table, page_table_stride, stream_block_table,
                         stream_table_stride, q, scale, out, lse, workspace, workspace_bytes, stream, true, first_blocks);
}

extern "C" padoc_status padoc_branch_decode_attn_e4m3(const padoc_kv_pool_e4m3 *pool, const padoc_decode_plan *info,
                                                      const int32_t *plan_dev, const int32_t *page_block_table,
                                                      int32_t page_table_stride, const int32_t *stream_block_table,
                                                      int32_t stream_table_stride, const void *q, float scale,
                                                      void *out, float *lse, void *workspace, size_t workspace_bytes,
                                                      padoc_stream_t stream)
{
    if (!pool || !info || !plan_dev || !q || !out || !lse) return PADOC_ERR_INVALID_ARGUMENT;
    const padoc_decode_config &cfg = info->cfg;
    if (pool->block_size != cfg.block_size || pool->num_kv_heads != cfg.num_kv_heads || pool->head_dim != cfg.head_dim)
        return PADOC_ERR_INVALID_ARGUMENT;
    if (!pool->k_codes || !pool->v_codes || !pool->k_scales || !pool->v_scales || pool->num_blocks < 1)
        return PADOC_ERR_INVALID_ARGUMENT;
    if (!(scale > 0.f) || !isfinite(scale)) return PADOC_ERR_INVALID_ARGUMENT;
    if (info->num_pages > 0 && (!page_block_table || page_table_stride < info->max_page_blocks))
        return PADOC_ERR_INVALID_ARGUMENT;
    if (info->num_streams > 0 && (!stream_block_table || stream_table_stride < info->max_stream_blocks))
        return PADOC_ERR_INVALID_ARGUMENT;
    if (info->num_streams == 0) return PADOC_OK;
    if ((((uintptr_t)pool->k_codes) | ((uintptr_t)pool->v_codes) | ((uintptr_t)q) | ((uintptr_t)out)) & 15)
        return PADOC_ERR_INVALID_ARGUMENT;
    if ((((uintptr_t)pool->k_scales) | ((uintptr_t)pool->v_scales)) & 3) return PADOC_ERR_INVALID_ARGUMENT;
    const DecodePool dp{true, pool->k_codes, pool->v_codes, pool->k_scales, pool->v_scales, pool->num_blocks};
    return decode_split_k(dp, info, plan_dev, page_block_table, page_table_stride, stream_block_table,
                          stream_table_stride, q, scale, out, lse, workspace, workspace_bytes, (cudaStream_t)stream);
}

extern "C" padoc_status padoc_launch_decode_step(const padoc_kv_pool *pool, const padoc_decode_plan *info,
                                                 const int32_t *stage, int64_t stage_words, int64_t off_page_table,
                                                 int32_t page_table_stride, int64_t off_stream_table,
                                                 int32_t stream_table_stride, int32_t *dev_ints,
                                                 int64_t dev_capacity_words, const void *q_host, void *q_dev,
                                                 float scale, void *out_dev, float *lse_dev, void *out_host,
                                                 float *lse_host, void *workspace, size_t workspace_bytes,
                                                 padoc_stream_t stream, padoc_stream_t copy_in,
                                                 padoc_stream_t copy_out, padoc_event_t ev_free, padoc_event_t ev_in,
                                                 padoc_event_t ev_dec)
{
    if (!pool || !info || !stage || !dev_ints || !q_host || !q_dev || !out_dev || !lse_dev || !out_host || !lse_host)
        return PADOC_ERR_INVALID_ARGUMENT;
    const bool piped = copy_in != nullptr;
    if (piped && (!copy_out || !ev_free || !ev_in || !ev_dec)) return PADOC_ERR_INVALID_ARGUMENT;
    const int64_t P = info->num_pages, S = info->num_streams;
    if (stage_words < info->plan_ints || dev_capacity_words < stage_words) return PADOC_ERR_INVALID_ARGUMENT;
    if ((((uintptr_t)dev_ints) & 255) || (off_page_table & 31) || (off_stream_table & 31)) return PADOC_ERR_INVALID_ARGUMENT;
    if (page_table_stride < 1 || stream_table_stride < 1) return PADOC_ERR_INVALID_ARGUMENT;
    if (off_page_table < info->plan_ints || off_page_table + P * page_table_stride > stage_words ||
        off_stream_table < info->plan_ints || off_stream_table + S * stream_table_stride > stage_words)
        return PADOC_ERR_INVALID_ARGUMENT;
    const bool overlap = off_page_table < off_stream_table ? off_page_table + P * page_table_stride > off_stream_table
                                                           : off_stream_table + S * stream_table_stride > off_page_table;
    if (P > 0 && S > 0 && overlap) return PADOC_ERR_INVALID_ARGUMENT;
    const size_t esz = pool->dtype == PADOC_DTYPE_BF16 ? 2 : 4;
    const size_t q_bytes = (size_t)S * info->cfg.num_q_heads * info->cfg.head_dim * esz;
    const size_t lse_bytes = (size_t)S * info->cfg.num_q_heads * sizeof(float);
    if (S == 0) return PADOC_OK;
    cudaStream_t cs = (cudaStream_t)stream;
    cudaStream_t cin = piped ? (cudaStream_t)copy_in : cs, cout = piped ? (cudaStream_t)copy_out : cs;
    // the step's integers and queries in (pinned host memory makes both copies asynchronous), once
    // this buffer set's previous step has copied its results out
    if (piped) PADOC_CUDA_TRY(cudaStreamWaitEvent(cin, (cudaEvent_t)ev_free, 0));
    PADOC_CUDA_TRY(cudaMemcpyAsync(dev_ints, stage, (size_t)stage_words * sizeof(int32_t), cudaMemcpyHostToDevice, cin));
    PADOC_CUDA_TRY(cudaMemcpyAsync(q_dev, q_host, q_bytes, cudaMemcpyHostToDevice, cin));
    if (piped) {
        PADOC_CUDA_TRY(cudaEventRecord((cudaEvent_t)ev_in, cin));
        PADOC_CUDA_TRY(cudaStreamWaitEvent(cs, (cudaEvent_t)ev_in, 0));
    }
    const padoc_status st = padoc_branch_decode_attn(pool, info, dev_ints, dev_ints + off_page_table, page_table_stride,
                                                     dev_ints + off_stream_table, stream_table_stride, q_dev, scale,
                                                     out_dev, lse_dev, workspace, workspace_bytes, stream);
    if (st != PADOC_OK) return st;
    // and the results out
    if (piped) {
        PADOC_CUDA_TRY(cudaEventRecord((cudaEvent_t)ev_dec, cs));
        PADOC_CUDA_TRY(cudaStreamWaitEvent(cout, (cudaEvent_t)ev_dec, 0));
    }
    PADOC_CUDA_TRY(cudaMemcpyAsync(out_host, out_dev, q_bytes, cudaMemcpyDeviceToHost, cout));
    PADOC_CUDA_TRY(cudaMemcpyAsync(lse_host, lse_dev, lse_bytes, cudaMemcpyDeviceToHost, cout));
    if (piped) PADOC_CUDA_TRY(cudaEventRecord((cudaEvent_t)ev_free, cout));
    return PADOC_OK;
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
