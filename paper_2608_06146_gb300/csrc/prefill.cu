// prefill.cu -- C3: packed variable-length ancestor prefill (App. C.1: one causal problem over
// the shared stream M and one bottom-right-aligned causal problem per branch over
// [K_{M<=f_k}; K_{Y_k}]), computed in packed order with no gather.
//
// The tile map lists, per 128-row q-tile, the 128-column k-tiles that hold a visible entry
// (fully masked tiles are never visited, as in Flex Attention's block mask) and whether every
// entry is visible (FULL: no masking) or not (PARTIAL: each row's two spans mask the tile).
//
// Warp-MMA kernel: one CTA per (q-tile, query head), 8 warps x 16 query rows, Q/K/V tiles staged
// by TMA (128-byte swizzle, 64-column panels), online softmax in registers (FlashAttention-2
// style), K/V double-buffered per k-tile.
#include <math.h>

#include "common.cuh"

namespace {

constexpr int kD = 128;
constexpr int kQT = PADOC_PREFILL_Q_TILE;   // 128 query rows per tile
constexpr int kKT = PADOC_PREFILL_K_TILE;   // 128 key columns per tile
constexpr int kPanel = kQT * 128;           // [128 rows][64 cols] bf16 = 16 KB
constexpr int kTileBytes = 2 * kPanel;      // two 64-column panels = 32 KB
constexpr int kKVStages = 2;
constexpr size_t kPrefillSmem = 1024 + kTileBytes /*Q*/ + (size_t)kKVStages * 2 * kTileBytes /*K,V*/ + 64;

struct PrefillParams {
    const int32_t *spans;
    const int32_t *row_ptr;
    const int32_t *tile_k;
    const int8_t *tile_kind;
    int64_t T;
    int32_t num_q_heads, num_kv_heads, num_q_tiles;
    float scale_log2;
    __nv_bfloat16 *out;
    float *lse;
    int *err;
};

__global__ void __launch_bounds__(256, 1)
prefill_mma_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                   const __grid_constant__ CUtensorMap vmap, const PrefillParams prm)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *sq = smem;
    uint8_t *skv = smem + kTileBytes;   // stage s: K at s*2*kTileBytes, V right after
    uint64_t *bars = (uint64_t *)(skv + (size_t)kKVStages * 2 * kTileBytes);   // [0] = Q, [1..] = KV

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int h = blockIdx.x;
    const int qt = prm.num_q_tiles - 1 - (int)blockIdx.y;   // heavier tiles (later in a page) first
    const int g = h / (prm.num_q_heads / prm.num_kv_heads);
    const int e0 = prm.row_ptr[qt], e1 = prm.row_ptr[qt + 1];
    const int ne = e1 - e0;

    if (tid == 0) {
        for (int i = 0; i < 1 + kKVStages; ++i) mbar_init(smem_u32(&bars[i]), 1);
        fence_barrier_init();
    }
    __syncthreads();

    auto issue_kv = [&](int e) {
        const int s = e % kKVStages;
        const uint32_t bar = smem_u32(&bars[1 + s]);
        const uint32_t kb = smem_u32(skv + (size_t)s * 2 * kTileBytes);
        const int kt = prm.tile_k[e0 + e];
        mbar_arrive_expect_tx(bar, 2 * kTileBytes);
        tma_load_2d(kb, &kmap, g * kD, kt * kKT, bar);
        tma_load_2d(kb + kPanel, &kmap, g * kD + 64, kt * kKT, bar);
        tma_load_2d(kb + kTileBytes, &vmap, g * kD, kt * kKT, bar);
        tma_load_2d(kb + kTileBytes + kPanel, &vmap, g * kD + 64, kt * kKT, bar);
    };
    if (tid == 0) {
        const uint32_t bar = smem_u32(&bars[0]);
        mbar_arrive_expect_tx(bar, kTileBytes);
        tma_load_2d(smem_u32(sq), &qmap, h * kD, qt * kQT, bar);
        tma_load_2d(smem_u32(sq) + kPanel, &qmap, h * kD + 64, qt * kQT, bar);
        for (int e = 0; e < kKVStages && e < ne; ++e) issue_kv(e);
    }

    // the two query rows of this thread and their spans
    const int64_t r0 = (int64_t)qt * kQT + warp * 16 + (lane >> 2), r1 = r0 + 8;
    int sp0[4] = {0, 0, 0, 0}, sp1[4] = {0, 0, 0, 0};
    if (r0 < prm.T) { const int4 v = *reinterpret_cast<const int4 *>(prm.spans + 4 * r0); sp0[0] = v.x; sp0[1] = v.y; sp0[2] = v.z; sp0[3] = v.w; }
    if (r1 < prm.T) { const int4 v = *reinterpret_cast<const int4 *>(prm.spans + 4 * r1); sp1[0] = v.x; sp1[1] = v.y; sp1[2] = v.z; sp1[3] = v.w; }

    bool ok = mbar_wait_bounded(smem_u32(&bars[0]), 0, prm.err, 10);
    if (__syncthreads_or(!ok)) {
        if (tid == 0)
            for (int e = 0; e < kKVStages && e < ne; ++e) mbar_wait_bounded(smem_u32(&bars[1 + e]), 0, prm.err, 11);
        return;
    }
    uint32_t qa[8][4];
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
        const uint32_t row = warp * 16 + (lane & 15);
        const uint32_t col = (ks & 3) * 16 + (lane >> 4) * 8;
        ldmatrix_x4(qa[ks], smem_u32(sq) + (ks >> 2) * kPanel + sw128_offset(row, col));
    }

    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    float o[16][4];
#pragma unroll
    for (int n = 0; n < 16; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;

    int e = 0;
    for (; e < ne; ++e) {
        const int s = e % kKVStages;
        ok = mbar_wait_bounded(smem_u32(&bars[1 + s]), (e / kKVStages) & 1, prm.err, 12);
        if (__syncthreads_or(!ok)) break;
        const int kt = prm.tile_k[e0 + e];
        const bool full = prm.tile_kind[e0 + e] == PADOC_TILE_FULL;
        const uint32_t kb = smem_u32(skv + (size_t)s * 2 * kTileBytes);
        const uint32_t vb = kb + kTileBytes;
#pragma unroll 1
        for (int sub = 0; sub < 2; ++sub) {   // 64-column halves of the k-tile
            float sc[8][4];
#pragma unroll
            for (int n = 0; n < 8; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
                for (int np = 0; np < 4; ++np) {
                    const int i = lane >> 3;
                    const uint32_t row = sub * 64 + np * 16 + (lane & 7) + (i >= 2 ? 8 : 0);
                    const uint32_t col = (ks & 3) * 16 + (i & 1) * 8;
                    uint32_t b[4];
                    ldmatrix_x4(b, kb + (ks >> 2) * kPanel + sw128_offset(row, col));
                    mma_bf16_16816(sc[2 * np], qa[ks], b[0], b[1]);
                    mma_bf16_16816(sc[2 * np + 1], qa[ks], b[2], b[3]);
                }
            }
            const int cbase = kt * kKT + sub * 64 + (lane & 3) * 2;
            float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
            for (int n = 0; n < 8; ++n) {
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    float v0 = sc[n][c] * prm.scale_log2, v1 = sc[n][2 + c] * prm.scale_log2;
                    if (!full) {
                        const int j = cbase + n * 8 + c;
                        const bool vis0 = (j >= sp0[0] && j < sp0[1]) || (j >= sp0[2] && j < sp0[3]);
                        const bool vis1 = (j >= sp1[0] && j < sp1[1]) || (j >= sp1[2] && j < sp1[3]);
                        v0 = vis0 ? v0 : -INFINITY;
                        v1 = vis1 ? v1 : -INFINITY;
                    }
                    sc[n][c] = v0; sc[n][2 + c] = v1;
                    mx0 = fmaxf(mx0, v0); mx1 = fmaxf(mx1, v1);
                }
            }
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
            const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
            const float al0 = mn0 == -INFINITY ? 1.f : fast_exp2(m0 - mn0);
            const float al1 = mn1 == -INFINITY ? 1.f : fast_exp2(m1 - mn1);
            const float b0 = mn0 == -INFINITY ? 0.f : mn0, b1 = mn1 == -INFINITY ? 0.f : mn1;
            m0 = mn0; m1 = mn1;
            float rs0 = 0.f, rs1 = 0.f;
            uint32_t pa[4][4];
#pragma unroll
            for (int n = 0; n < 8; ++n) {
                const float p00 = fast_exp2(sc[n][0] - b0), p01 = fast_exp2(sc[n][1] - b0);
                const float p10 = fast_exp2(sc[n][2] - b1), p11 = fast_exp2(sc[n][3] - b1);
                rs0 += p00 + p01; rs1 += p10 + p11;
                pa[n >> 1][(n & 1) * 2 + 0] = pack_bf16x2(p00, p01);
                pa[n >> 1][(n & 1) * 2 + 1] = pack_bf16x2(p10, p11);
            }
            l0 = l0 * al0 + rs0;
            l1 = l1 * al1 + rs1;
#pragma unroll
            for (int n = 0; n < 16; ++n) { o[n][0] *= al0; o[n][1] *= al0; o[n][2] *= al1; o[n][3] *= al1; }
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
                // A fragment order: a0 (rows 0-7, keys 0-7), a1 (rows 8-15, keys 0-7),
                //                   a2 (rows 0-7, keys 8-15), a3 (rows 8-15, keys 8-15)
                uint32_t a[4] = {pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3]};
#pragma unroll
                for (int np = 0; np < 8; ++np) {
                    const int i = lane >> 3;
                    const uint32_t row = sub * 64 + kk * 16 + (lane & 7) + ((i & 1) ? 8 : 0);
                    const uint32_t colg = np * 16 + (i >> 1) * 8;   // dims 0..127
                    uint32_t b[4];
                    ldmatrix_x4_trans(b, vb + (colg >> 6) * kPanel + sw128_offset(row, colg & 63));
                    mma_bf16_16816(o[2 * np], a, b[0], b[1]);
                    mma_bf16_16816(o[2 * np + 1], a, b[2], b[3]);
                }
            }
        }
        __syncthreads();
        if (tid == 0 && e + kKVStages < ne) issue_kv(e + kKVStages);
    }
    if (e < ne) {   // a wait ran out: let issued copies land, then leave
        if (tid == 0)
            for (int r = e + 1; r < ne && r < e + kKVStages; ++r)
                mbar_wait_bounded(smem_u32(&bars[1 + r % kKVStages]), (r / kKVStages) & 1, prm.err, 13);
        return;
    }

    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
    const float inv0 = l0 > 0.f ? 1.f / l0 : 0.f, inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
#pragma unroll
    for (int n = 0; n < 16; ++n) {
        const int dcol = n * 8 + (lane & 3) * 2;
        if (r0 < prm.T)
            *reinterpret_cast<uint32_t *>(prm.out + ((size_t)r0 * prm.num_q_heads + h) * kD + dcol) =
                pack_bf16x2(o[n][0] * inv0, o[n][1] * inv0);
        if (r1 < prm.T)
            *reinterpret_cast<uint32_t *>(prm.out + ((size_t)r1 * prm.num_q_heads + h) * kD + dcol) =
                pack_bf16x2(o[n][2] * inv1, o[n][3] * inv1);
    }
    if ((lane & 3) == 0) {
        if (r0 < prm.T) prm.lse[(size_t)r0 * prm.num_q_heads + h] = l0 > 0.f ? (m0 + log2f(l0)) * PADOC_LN2 : -INFINITY;
        if (r1 < prm.T) prm.lse[(size_t)r1 * prm.num_q_heads + h] = l1 > 0.f ? (m1 + log2f(l1)) * PADOC_LN2 : -INFINITY;
    }
}

// fp32 bring-up path: one warp per (token, query head) over its two spans, keys in order.
template <int D>
__global__ void __launch_bounds__(128) prefill_f32_kernel(const float *__restrict__ q, const float *__restrict__ k,
                                                          const float *__restrict__ v, const int32_t *__restrict__ spans,
                                                          int64_t T, int32_t hq, int32_t hkv, float scale_log2,
                                                          float *__restrict__ out, float *__restrict__ lse)
{
    constexpr int E = D / 32;
    const int64_t row = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= T * hq) return;
    const int64_t t = row / hq;
    const int h = (int)(row % hq), g = h / (hq / hkv);
    float qv[E], ov[E];
#pragma unroll
    for (int e = 0; e < E; ++e) { qv[e] = q[row * D + lane + 32 * e]; ov[e] = 0.f; }
    float m = -INFINITY, l = 0.f;
    for (int sidx = 0; sidx < 2; ++sidx) {
        const int a = spans[4 * t + 2 * sidx], b = spans[4 * t + 2 * sidx + 1];
        for (int j = a; j < b; ++j) {
            const size_t kr = ((size_t)j * hkv + g) * D;
            float dot = 0.f;
#pragma unroll
            for (int e = 0; e < E; ++e) dot = fmaf(qv[e], k[kr + lane + 32 * e], dot);
#pragma unroll
            for (int sh = 16; sh > 0; sh >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, sh);
            const float sc = dot * scale_log2;
            const float mn = fmaxf(m, sc);
            const float al = exp2f(m - mn), p = exp2f(sc - mn);
            l = l * al + p;
#pragma unroll
            for (int e = 0; e < E; ++e) ov[e] = fmaf(p, v[kr + lane + 32 * e], ov[e] * al);
            m = mn;
        }
    }
    const bool empty = !(l > 0.f);
#pragma unroll
    for (int e = 0; e < E; ++e) out[row * D + lane + 32 * e] = empty ? 0.f : ov[e] / l;
    if (lane == 0) lse[row] = empty ? -INFINITY : (m + log2f(l)) * PADOC_LN2;
}

}  // namespace

extern "C" padoc_status padoc_ancestor_prefill_attn(const void *q, const void *k, const void *v, padoc_dtype dtype,
                                                    int64_t total_tokens, int32_t num_q_heads, int32_t num_kv_heads,
                                                    int32_t head_dim, const int32_t *spans_dev,
                                                    const int32_t *tile_row_ptr_dev, const int32_t *tile_k_dev,
                                                    const int8_t *tile_kind_dev, int32_t q_tile, int32_t k_tile,
                                                    float scale, void *out, float *lse, padoc_stream_t stream)
{
    if (total_tokens < 0 || total_tokens >= INT32_MAX) return PADOC_ERR_INVALID_ARGUMENT;
    if (num_q_heads < 1 || num_kv_heads < 1 || num_q_heads % num_kv_heads != 0) return PADOC_ERR_INVALID_ARGUMENT;
    if (!(scale > 0.f) || !isfinite(scale)) return PADOC_ERR_INVALID_ARGUMENT;
    if (total_tokens == 0) return PADOC_OK;
    if (!q || !k || !v || !spans_dev || !out || !lse) return PADOC_ERR_INVALID_ARGUMENT;
    if ((((uintptr_t)q) | ((uintptr_t)k) | ((uintptr_t)v) | ((uintptr_t)out) | ((uintptr_t)spans_dev)) & 15)
        return PADOC_ERR_INVALID_ARGUMENT;
    cudaStream_t cs = (cudaStream_t)stream;
    const float sl2 = scale * PADOC_LOG2E;
    if (dtype == PADOC_DTYPE_F32) {
        if (head_dim != 64 && head_dim != 128) return PADOC_ERR_UNSUPPORTED;
        const int64_t rows = total_tokens * num_q_heads;
        const unsigned grid = (unsigned)((rows + 3) / 4);
        if (head_dim == 64)
            prefill_f32_kernel<64><<<grid, 128, 0, cs>>>((const float *)q, (const float *)k, (const float *)v, spans_dev,
                                                         total_tokens, num_q_heads, num_kv_heads, sl2, (float *)out, lse);
        else
            prefill_f32_kernel<128><<<grid, 128, 0, cs>>>((const float *)q, (const float *)k, (const float *)v, spans_dev,
                                                          total_tokens, num_q_heads, num_kv_heads, sl2, (float *)out, lse);
        return padoc_launch_status();
    }
    if (dtype != PADOC_DTYPE_BF16) return PADOC_ERR_UNSUPPORTED;
    if (head_dim != kD) return PADOC_ERR_UNSUPPORTED;
    if (q_tile != kQT || k_tile != kKT) return PADOC_ERR_INVALID_ARGUMENT;
    if (!tile_row_ptr_dev || !tile_k_dev || !tile_kind_dev) return PADOC_ERR_INVALID_ARGUMENT;
    return padoc_launch_prefill_tc(q, k, v, total_tokens, num_q_heads, num_kv_heads, spans_dev, tile_row_ptr_dev,
                                   tile_k_dev, tile_kind_dev, sl2, out, lse, cs);
}
