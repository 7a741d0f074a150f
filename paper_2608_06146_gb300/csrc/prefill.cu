// prefill.cu -- C3: packed variable-length ancestor prefill (App. C.1: one causal problem over
// the shared stream M and one bottom-right-aligned causal problem per branch over
// [K_{M<=f_k}; K_{Y_k}]), computed in packed order with no gather.
//
// The tile map lists, per 128-row q-tile, the 128-column k-tiles that hold a visible entry
// (fully masked tiles are never visited, as in Flex Attention's block mask) and whether every
// entry is visible (FULL: no masking) or not (PARTIAL: each row's two spans mask the tile).
//
// The bf16 path runs on the tensor cores (prefill_tc.cu); this file holds the host entry point,
// its validation and the fp32 bring-up kernel.
#include <math.h>

#include "common.cuh"

namespace {

constexpr int kD = 128;

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
    if (q_tile != PADOC_PREFILL_Q_TILE || k_tile != PADOC_PREFILL_K_TILE) return PADOC_ERR_INVALID_ARGUMENT;
    if (!tile_row_ptr_dev || !tile_k_dev || !tile_kind_dev) return PADOC_ERR_INVALID_ARGUMENT;
    return padoc_launch_prefill_tc(q, k, v, total_tokens, num_q_heads, num_kv_heads, spans_dev, tile_row_ptr_dev,
                                   tile_k_dev, tile_kind_dev, sl2, out, lse, cs);
}
