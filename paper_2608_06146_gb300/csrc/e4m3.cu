// e4m3.cu -- writing the FP8 (E4M3) variant of the paged KV cache (C5): whole blocks quantized at
// once (a page's prefix after its prefill), and one row per input appended by a decoding loop
// (Algorithm 1's "Append i to the cache", App. E.1). The paper serves a bf16 cache; this variant
// stores K and V as E4M3 codes with one fp32 scale per (block, KV head), the scale being amax / 448
// over the rows the block holds, so that a block's largest magnitude maps to the format's largest
// finite value. All arithmetic that decides a code is fp32 with round-to-nearest-even (division and
// product rounded once each), so the codes are a function of the inputs alone.
#include "common.cuh"

namespace {

constexpr int kD = 128;        // head_dim of the E4M3 path
constexpr int kBlk = 16;       // tokens per block
constexpr int kThreads = 128;  // one thread per dim of a row (append), 16 values each (quantize)

__device__ __forceinline__ float block_max128(float v, float *red)
{
#pragma unroll
    for (int sh = 16; sh > 0; sh >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, sh));
    const int warp = threadIdx.x >> 5;
    __syncthreads();   // red may still be read by a previous reduction
    if ((threadIdx.x & 31) == 0) red[warp] = v;
    __syncthreads();
    return fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
}

// Grid (count, Hkv, 2 = K / V): (source block i, head g) of k_src or v_src ([count][Hkv][16][128]
// bf16) becomes (block dst_blocks[i], head g) of the pool: scale = amax / 448, codes of x / scale
// (0 and codes 0 for an all-zero one). Thread t converts row t / 8, dims 16 (t % 8) .. + 15.
__global__ void __launch_bounds__(kThreads) quantize_blocks_kernel(const __nv_bfloat16 *__restrict__ k_src,
                                                                   const __nv_bfloat16 *__restrict__ v_src,
                                                                   const int32_t *__restrict__ dst_blocks,
                                                                   uint8_t *__restrict__ k_codes, uint8_t *__restrict__ v_codes,
                                                                   float *__restrict__ k_scales, float *__restrict__ v_scales,
                                                                   int32_t num_blocks, int32_t hkv, int *err)
{
    __shared__ float red[4];
    const int i = blockIdx.x, g = blockIdx.y;
    const bool is_v = blockIdx.z != 0;
    const int32_t b = dst_blocks[i];
    if (b < 0 || b >= num_blocks) {
        if (threadIdx.x == 0 && g == 0 && !is_v) padoc_record_error(err, PADOC_DEVERR_BLOCK_ID, b);
        return;
    }
    const __nv_bfloat16 *src = (is_v ? v_src : k_src) + ((size_t)i * hkv + g) * kBlk * kD + threadIdx.x * 16;
    const uint4 u0 = reinterpret_cast<const uint4 *>(src)[0], u1 = reinterpret_cast<const uint4 *>(src)[1];
    const uint32_t w[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
    float x[16];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        x[2 * k] = __uint_as_float(w[k] << 16);
        x[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
    }
    float a = 0.f;
#pragma unroll
    for (int k = 0; k < 16; ++k) a = fmaxf(a, fabsf(x[k]));
    a = block_max128(a, red);
    const float s = __fdiv_rn(a, 448.f);
    uint32_t o[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        uint16_t lo = 0, hi = 0;
        if (s > 0.f) {
            lo = f32x2_to_e4m3x2(__fdiv_rn(x[4 * k], s), __fdiv_rn(x[4 * k + 1], s));
            hi = f32x2_to_e4m3x2(__fdiv_rn(x[4 * k + 2], s), __fdiv_rn(x[4 * k + 3], s));
        }
        o[k] = (uint32_t)lo | ((uint32_t)hi << 16);
    }
    uint8_t *dst = (is_v ? v_codes : k_codes) + ((size_t)b * hkv + g) * kBlk * kD + threadIdx.x * 16;
    *reinterpret_cast<uint4 *>(dst) = make_uint4(o[0], o[1], o[2], o[3]);
    if (threadIdx.x == 0) (is_v ? v_scales : k_scales)[(size_t)b * hkv + g] = s;
}

// One CTA per input i: its K and V rows (row src_rows[i] of k_src / v_src, [src_total][Hkv][128]
// bf16) go to row r = slots[i] % 16 of block slots[i] / 16, every KV head, by the scale rule: the
// new scale is max(old, amax(row) / 448) (the old one taken as 0 at r = 0, which starts a block
// afresh); when it grows from a nonzero old scale, rows 0 .. r-1 are re-encoded (code value x old
// scale, then / new scale, each rounded to fp32); the row's codes are those of x / new scale. The
// query row goes to row i of q_dst. Thread t owns dim t.
__global__ void __launch_bounds__(kThreads) append_e4m3_kernel(const __nv_bfloat16 *__restrict__ k_src,
                                                               const __nv_bfloat16 *__restrict__ v_src,
                                                               const uint4 *__restrict__ q_src, int64_t src_total,
                                                               uint4 *__restrict__ q_dst, const int32_t *__restrict__ src_rows,
                                                               const int32_t *__restrict__ slots, uint8_t *__restrict__ k_codes,
                                                               uint8_t *__restrict__ v_codes, float *__restrict__ k_scales,
                                                               float *__restrict__ v_scales, int64_t pool_slots, int32_t hkv,
                                                               int32_t hq, int *err)
{
    __shared__ float red[4];
    // a programmatic dependent of the previous kernel in the stream, as the bf16 append
    pdl_wait_prerequisite();
    pdl_launch_dependents();
    const int64_t i = blockIdx.x;
    const int64_t row = src_rows ? (int64_t)src_rows[i] : i;
    const int64_t slot = slots[i];
    if (slot < 0 || slot >= pool_slots || row < 0 || row >= src_total) {
        if (threadIdx.x == 0)
            padoc_record_error(err, PADOC_DEVERR_BLOCK_ID, (slot < 0 || slot >= pool_slots) ? (int)slot : (int)row);
        return;
    }
    const int64_t blk = slot / kBlk;
    const int r = (int)(slot % kBlk);
    const int t = threadIdx.x;
    for (int u = 0; u < 2 * hkv; ++u) {
        const bool is_v = u >= hkv;
        const int g = is_v ? u - hkv : u;
        const float x = __bfloat162float((is_v ? v_src : k_src)[(row * hkv + g) * kD + t]);
        const float a = block_max128(fabsf(x), red);
        float *scp = (is_v ? v_scales : k_scales) + blk * hkv + g;
        const float s_old = r == 0 ? 0.f : *scp;
        const float cand = __fdiv_rn(a, 448.f);
        const float s_new = cand > s_old ? cand : s_old;
        uint8_t *codes = (is_v ? v_codes : k_codes) + (blk * hkv + g) * kBlk * kD;
        if (s_new > s_old && s_old > 0.f)
            for (int rr = 0; rr < r; ++rr) {
                const float y = __fmul_rn(e4m3_to_f32(codes[rr * kD + t]), s_old);
                codes[rr * kD + t] = (uint8_t)(f32x2_to_e4m3x2(__fdiv_rn(y, s_new), 0.f) & 0xFF);
            }
        codes[r * kD + t] = s_new > 0.f ? (uint8_t)(f32x2_to_e4m3x2(__fdiv_rn(x, s_new), 0.f) & 0xFF) : (uint8_t)0;
        __syncthreads();   // every thread has read the old scale before it is replaced
        if (t == 0) *scp = s_new;
    }
    if (q_src) {
        const int q_vecs = hq * (kD * 2 / 16);
        const uint4 *qs = q_src + row * q_vecs;
        uint4 *qd = q_dst + i * q_vecs;
        for (int c = t; c < q_vecs; c += kThreads) qd[c] = qs[c];
    }
}

bool e4m3_pool_ok(const padoc_kv_pool_e4m3 *pool)
{
    return pool && pool->k_codes && pool->v_codes && pool->k_scales && pool->v_scales && pool->num_blocks >= 1 &&
           pool->num_kv_heads >= 1 && pool->block_size >= 1 && pool->head_dim >= 1;
}

}  // namespace

extern "C" padoc_status padoc_quantize_kv_blocks(const padoc_kv_pool_e4m3 *pool, const void *k_src, const void *v_src,
                                                 const int32_t *dst_blocks, int32_t count, padoc_stream_t stream)
{
    if (!e4m3_pool_ok(pool) || count < 0) return PADOC_ERR_INVALID_ARGUMENT;
    if (pool->block_size != kBlk || pool->head_dim != kD || pool->num_kv_heads > 65535) return PADOC_ERR_UNSUPPORTED;
    if (count == 0) return PADOC_OK;
    if (!k_src || !v_src || !dst_blocks) return PADOC_ERR_INVALID_ARGUMENT;
    const uintptr_t align = (uintptr_t)pool->k_codes | (uintptr_t)pool->v_codes | (uintptr_t)k_src | (uintptr_t)v_src;
    if ((align & 15) || (((uintptr_t)pool->k_scales | (uintptr_t)pool->v_scales) & 3)) return PADOC_ERR_INVALID_ARGUMENT;
    int *err = padoc_device_error_word();
    if (!err) return PADOC_ERR_CUDA;
    quantize_blocks_kernel<<<dim3((unsigned)count, (unsigned)pool->num_kv_heads, 2), kThreads, 0, (cudaStream_t)stream>>>(
        (const __nv_bfloat16 *)k_src, (const __nv_bfloat16 *)v_src, dst_blocks, (uint8_t *)pool->k_codes,
        (uint8_t *)pool->v_codes, (float *)pool->k_scales, (float *)pool->v_scales, pool->num_blocks, pool->num_kv_heads,
        err);
    return padoc_launch_status();
}

extern "C" padoc_status padoc_append_inputs_e4m3(const padoc_kv_pool_e4m3 *pool, const void *k_src, const void *v_src,
                                                 const void *q_src, int64_t src_total, int32_t num_q_heads, void *q_dst,
                                                 const int32_t *src_rows, const int32_t *slots, int32_t count,
                                                 padoc_stream_t stream)
{
    if (!e4m3_pool_ok(pool) || count < 0 || src_total < 0) return PADOC_ERR_INVALID_ARGUMENT;
    if (pool->block_size != kBlk || pool->head_dim != kD) return PADOC_ERR_UNSUPPORTED;
    if (count == 0) return PADOC_OK;
    if (!k_src || !v_src || !slots) return PADOC_ERR_INVALID_ARGUMENT;
    if (q_src && (!q_dst || num_q_heads < 1)) return PADOC_ERR_INVALID_ARGUMENT;
    const uintptr_t align = (uintptr_t)k_src | (uintptr_t)v_src | (uintptr_t)q_src | (uintptr_t)q_dst;
    if ((align & 15) || (((uintptr_t)pool->k_scales | (uintptr_t)pool->v_scales) & 3)) return PADOC_ERR_INVALID_ARGUMENT;
    int *err = padoc_device_error_word();
    if (!err) return PADOC_ERR_CUDA;
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3((unsigned)count);
    lc.blockDim = dim3(kThreads);
    lc.stream = (cudaStream_t)stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // see the kernel's wait
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = 1;
    PADOC_CUDA_TRY(cudaLaunchKernelEx(&lc, append_e4m3_kernel, (const __nv_bfloat16 *)k_src, (const __nv_bfloat16 *)v_src,
                                      (const uint4 *)q_src, src_total, (uint4 *)q_dst, src_rows, slots,
                                      (uint8_t *)pool->k_codes, (uint8_t *)pool->v_codes, (float *)pool->k_scales,
                                      (float *)pool->v_scales, (int64_t)pool->num_blocks * kBlk, pool->num_kv_heads,
                                      q_src ? num_q_heads : 0, err));
    return padoc_launch_status();
}
