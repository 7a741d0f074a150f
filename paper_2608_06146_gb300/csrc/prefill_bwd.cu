// prefill_bwd.cu -- gradients of C3, the packed ancestor prefill (App. C.1: training through the
// tree-varlen attention; Sec. 3.2 visibility): the host entry point, its validation and the fp32
// bring-up kernels (a per-row statistics pass, dQ and dK/dV). The bf16 passes run on the tensor
// cores (prefill_bwd_tc.cu).
//
// Per query row and head the backward needs lse (from the forward) and D = sum_c dO[c] O[c]
// (the softmax's chain-rule term, equal to sum_j P_j dP_j). Both paths write, per head,
// [Hq][t_pad] with t_pad = ceil(T / 128) * 128, the negated base-2 log-sum-exp -lse2 (so that
// P = exp2(S c + (-lse2)) is one fused multiply-add and an exponential) and D; padded rows hold
// -lse2 = -inf and D = 0, so that their P is exactly 0 and the tile passes need no row test.
#include <math.h>

#include "common.cuh"

namespace {

constexpr int64_t kPad = 128;

// fp32 path: one warp per (row, head): D = dO . O and -lse * log2(e), transposed to [Hq][t_pad].
// (The bf16 path computes both inside its dQ pass.)
template <int D>
__global__ void __launch_bounds__(256) prefill_bwd_stats_kernel(const float *__restrict__ out, const float *__restrict__ dout,
                                                                const float *__restrict__ lse, int64_t total_tokens,
                                                                int64_t t_pad, int32_t hq, float *__restrict__ lt,
                                                                float *__restrict__ dt)
{
    constexpr int E = D / 32;
    const int64_t r = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (r >= t_pad * hq) return;
    const int64_t t = r / hq;
    const int h = (int)(r % hq);
    float acc = 0.f;
    if (t < total_tokens) {
        const float *o = out + r * D + lane * E;
        const float *g = dout + r * D + lane * E;
#pragma unroll
        for (int e = 0; e < E; ++e) acc = fmaf(o[e], g[e], acc);
#pragma unroll
        for (int sh = 16; sh > 0; sh >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, sh);
    }
    if (lane == 0) {
        const size_t w = (size_t)h * t_pad + t;
        if (t < total_tokens) {
            const float l = lse[r];
            lt[w] = l == -INFINITY ? -INFINITY : -l * PADOC_LOG2E;   // a row that sees nothing has P = 0
            dt[w] = acc;
        } else {
            lt[w] = -INFINITY;
            dt[w] = 0.f;
        }
    }
}

// fp32 bring-up, dQ: one warp per (row, head) over its two spans, keys in order.
template <int D>
__global__ void __launch_bounds__(128) prefill_bwd_dq_f32_kernel(const float *__restrict__ q, const float *__restrict__ k,
                                                                 const float *__restrict__ v, const float *__restrict__ dout,
                                                                 const int32_t *__restrict__ spans, const float *__restrict__ lt,
                                                                 const float *__restrict__ dt, int64_t total_tokens,
                                                                 int64_t t_pad, int32_t hq, int32_t hkv, float c,
                                                                 float scale, float *__restrict__ dq)
{
    constexpr int E = D / 32;
    const int64_t r = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (r >= total_tokens * hq) return;
    const int64_t t = r / hq;
    const int h = (int)(r % hq), g = h / (hq / hkv);
    const float l2 = lt[(size_t)h * t_pad + t], dd = dt[(size_t)h * t_pad + t];
    float qv[E], gv[E], acc[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
        qv[e] = q[r * D + lane + 32 * e];
        gv[e] = dout[r * D + lane + 32 * e];
        acc[e] = 0.f;
    }
    for (int sidx = 0; sidx < 2; ++sidx) {
        const int a = spans[4 * t + 2 * sidx], b = spans[4 * t + 2 * sidx + 1];
        for (int j = a; j < b; ++j) {
            const size_t kr = ((size_t)j * hkv + g) * D;
            float s = 0.f, dp = 0.f;
#pragma unroll
            for (int e = 0; e < E; ++e) {
                s = fmaf(qv[e], k[kr + lane + 32 * e], s);
                dp = fmaf(gv[e], v[kr + lane + 32 * e], dp);
            }
#pragma unroll
            for (int sh = 16; sh > 0; sh >>= 1) {
                s += __shfl_xor_sync(0xffffffffu, s, sh);
                dp += __shfl_xor_sync(0xffffffffu, dp, sh);
            }
            const float ds = exp2f(fmaf(s, c, l2)) * (dp - dd);
#pragma unroll
            for (int e = 0; e < E; ++e) acc[e] = fmaf(ds, k[kr + lane + 32 * e], acc[e]);
        }
    }
#pragma unroll
    for (int e = 0; e < E; ++e) dq[r * D + lane + 32 * e] = acc[e] * scale;
}

// fp32 bring-up, dK/dV: one warp per (key, KV head) over the queries of the q-tiles the key-major
// map lists for the key's k-tile, each tested against its two spans.
template <int D>
__global__ void __launch_bounds__(128) prefill_bwd_dkv_f32_kernel(
    const float *__restrict__ q, const float *__restrict__ k, const float *__restrict__ v, const float *__restrict__ dout,
    const int32_t *__restrict__ spans, const float *__restrict__ lt, const float *__restrict__ dt,
    const int32_t *__restrict__ col_ptr, const int32_t *__restrict__ q_tiles, int32_t q_tile, int32_t k_tile,
    int64_t total_tokens, int64_t t_pad, int32_t hq, int32_t hkv, float c, float scale, float *__restrict__ dk,
    float *__restrict__ dv)
{
    constexpr int E = D / 32;
    const int64_t r = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (r >= total_tokens * hkv) return;
    const int64_t j = r / hkv;
    const int g = (int)(r % hkv), group = hq / hkv;
    const int kt = (int)(j / k_tile);
    float kv[E], vv[E], ak[E], av[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
        kv[e] = k[r * D + lane + 32 * e];
        vv[e] = v[r * D + lane + 32 * e];
        ak[e] = 0.f;
        av[e] = 0.f;
    }
    for (int en = col_ptr[kt]; en < col_ptr[kt + 1]; ++en) {
        const int64_t i0 = (int64_t)q_tiles[en] * q_tile;
        const int64_t i1 = i0 + q_tile < total_tokens ? i0 + q_tile : total_tokens;
        for (int64_t i = i0; i < i1; ++i) {
            const int4 w = *reinterpret_cast<const int4 *>(spans + 4 * i);
            if (!((j >= w.x && j < w.y) || (j >= w.z && j < w.w))) continue;
            for (int h = g * group; h < (g + 1) * group; ++h) {
                const size_t qr = ((size_t)i * hq + h) * D;
                float s = 0.f, dp = 0.f;
#pragma unroll
                for (int e = 0; e < E; ++e) {
                    s = fmaf(q[qr + lane + 32 * e], kv[e], s);
                    dp = fmaf(dout[qr + lane + 32 * e], vv[e], dp);
                }
#pragma unroll
                for (int sh = 16; sh > 0; sh >>= 1) {
                    s += __shfl_xor_sync(0xffffffffu, s, sh);
                    dp += __shfl_xor_sync(0xffffffffu, dp, sh);
                }
                const float p = exp2f(fmaf(s, c, lt[(size_t)h * t_pad + i]));
                const float ds = p * (dp - dt[(size_t)h * t_pad + i]);
#pragma unroll
                for (int e = 0; e < E; ++e) {
                    ak[e] = fmaf(ds, q[qr + lane + 32 * e], ak[e]);
                    av[e] = fmaf(p, dout[qr + lane + 32 * e], av[e]);
                }
            }
        }
    }
#pragma unroll
    for (int e = 0; e < E; ++e) {
        dk[r * D + lane + 32 * e] = ak[e] * scale;
        dv[r * D + lane + 32 * e] = av[e];
    }
}

int64_t pad_rows(int64_t T) { return (T + kPad - 1) / kPad * kPad; }

bool map_ok(const padoc_tile_map_dev *m, bool key_major, int32_t q_tile, int32_t k_tile)
{
    return m && m->ptr && m->idx && m->kind && (!key_major || m->order) && m->q_tile == q_tile && m->k_tile == k_tile;
}

}  // namespace

extern "C" padoc_status padoc_prefill_bwd_workspace_size(int64_t total_tokens, int32_t num_q_heads, size_t *bytes)
{
    if (!bytes || total_tokens < 0 || total_tokens >= INT32_MAX || num_q_heads < 1) return PADOC_ERR_INVALID_ARGUMENT;
    // -lse2 and D per head, then the split dK/dV units' fp32 partials: at most ceil(T / 128) units,
    // each two halves x (dV, dK) x 128 keys x 128 dims
    *bytes = 2 * (size_t)num_q_heads * (size_t)pad_rows(total_tokens) * sizeof(float) +
             (size_t)pad_rows(total_tokens) * PADOC_BWD_SPLIT_BYTES_PER_TOKEN;
    return PADOC_OK;
}

extern "C" padoc_status padoc_ancestor_prefill_bwd(const void *q, const void *k, const void *v, const void *out,
                                                   const void *dout, const float *lse, padoc_dtype dtype,
                                                   int64_t total_tokens, int32_t num_q_heads, int32_t num_kv_heads,
                                                   int32_t head_dim, const int32_t *spans_dev,
                                                   const padoc_tile_map_dev *q_map, const padoc_tile_map_dev *k_map,
                                                   float scale, void *dq, void *dk, void *dv, void *workspace,
                                                   size_t workspace_bytes, padoc_stream_t stream)
{
    if (total_tokens < 0 || total_tokens >= INT32_MAX) return PADOC_ERR_INVALID_ARGUMENT;
    if (num_q_heads < 1 || num_kv_heads < 1 || num_q_heads % num_kv_heads != 0) return PADOC_ERR_INVALID_ARGUMENT;
    if (!(scale > 0.f) || !isfinite(scale)) return PADOC_ERR_INVALID_ARGUMENT;
    if (dtype != PADOC_DTYPE_F32 && dtype != PADOC_DTYPE_BF16) return PADOC_ERR_UNSUPPORTED;
    if (dtype == PADOC_DTYPE_BF16 ? head_dim != 128 : (head_dim != 64 && head_dim != 128)) return PADOC_ERR_UNSUPPORTED;
    if (total_tokens == 0) return PADOC_OK;
    if (!q || !k || !v || !out || !dout || !lse || !spans_dev || !dq || !dk || !dv || !workspace)
        return PADOC_ERR_INVALID_ARGUMENT;
    if ((((uintptr_t)q) | ((uintptr_t)k) | ((uintptr_t)v) | ((uintptr_t)out) | ((uintptr_t)dout) | ((uintptr_t)dq) |
         ((uintptr_t)dk) | ((uintptr_t)dv) | ((uintptr_t)spans_dev)) & 15)
        return PADOC_ERR_INVALID_ARGUMENT;
    if (((uintptr_t)workspace) & 255) return PADOC_ERR_INVALID_ARGUMENT;
    if (!map_ok(q_map, false, PADOC_BWD_DQ_Q_TILE, PADOC_BWD_DQ_K_TILE) ||
        !map_ok(k_map, true, PADOC_BWD_DKV_Q_TILE, PADOC_BWD_DKV_K_TILE))
        return PADOC_ERR_INVALID_ARGUMENT;
    size_t need = 0;
    padoc_prefill_bwd_workspace_size(total_tokens, num_q_heads, &need);
    if (workspace_bytes < need) return PADOC_ERR_WORKSPACE_TOO_SMALL;

    cudaStream_t cs = (cudaStream_t)stream;
    const int64_t T = total_tokens, t_pad = pad_rows(T);
    float *lt = (float *)workspace;
    float *dt = lt + (size_t)num_q_heads * t_pad;
    float *split = dt + (size_t)num_q_heads * t_pad;   // the split dK/dV units' partials
    const float c = scale * PADOC_LOG2E;
    const unsigned sgrid = (unsigned)((t_pad * num_q_heads + 7) / 8);
    if (dtype == PADOC_DTYPE_BF16)   // the tensor-core dQ pass computes the statistics itself
        return padoc_launch_prefill_bwd_tc(q, k, v, out, dout, lse, T, num_q_heads, num_kv_heads, spans_dev, q_map,
                                           k_map, lt, dt, split, t_pad, scale, dq, dk, dv, cs);
    const unsigned qgrid = (unsigned)((T * num_q_heads + 3) / 4), kgrid = (unsigned)((T * num_kv_heads + 3) / 4);
#define PADOC_BWD_F32(D)                                                                                              \
    do {                                                                                                              \
        prefill_bwd_stats_kernel<D><<<sgrid, 256, 0, cs>>>((const float *)out, (const float *)dout, lse, T,    \
                                                                  t_pad, num_q_heads, lt, dt);                        \
        prefill_bwd_dq_f32_kernel<D><<<qgrid, 128, 0, cs>>>((const float *)q, (const float *)k, (const float *)v,     \
                                                            (const float *)dout, spans_dev, lt, dt, T, t_pad,          \
                                                            num_q_heads, num_kv_heads, c, scale, (float *)dq);         \
        prefill_bwd_dkv_f32_kernel<D><<<kgrid, 128, 0, cs>>>(                                                         \
            (const float *)q, (const float *)k, (const float *)v, (const float *)dout, spans_dev, lt, dt, k_map->ptr, \
            k_map->idx, k_map->q_tile, k_map->k_tile, T, t_pad, num_q_heads, num_kv_heads, c, scale, (float *)dk,     \
            (float *)dv);                                                                                             \
    } while (0)
    if (head_dim == 64)
        PADOC_BWD_F32(64);
    else
        PADOC_BWD_F32(128);
#undef PADOC_BWD_F32
    return padoc_launch_status();
}
