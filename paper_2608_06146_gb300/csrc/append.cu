// append.cu -- Algorithm 1's append ("Append i to the cache", App. E.1) into the paged pool (C5):
// the K and V rows of one input per live stream go to the slot the scheduler gave it, and the
// inputs' queries are laid out in the decode call's stream order. Also used for a new page's prefix.
//
// One CTA per input; the pool keeps a (block, KV head) as block_size contiguous rows, so a token's
// head rows are head_dim-wide runs at stride block_size * head_dim. Every copy is 16-byte vectors.
#include "common.cuh"

namespace {

constexpr int kThreads = 128;

__global__ void __launch_bounds__(kThreads) append_kernel(const uint4 *__restrict__ k_src, const uint4 *__restrict__ v_src,
                                                          const uint4 *__restrict__ q_src, int64_t src_total,
                                                          uint4 *__restrict__ q_dst, const int32_t *__restrict__ src_rows,
                                                          const int32_t *__restrict__ slots, uint4 *__restrict__ k_pool,
                                                          uint4 *__restrict__ v_pool, int64_t pool_slots,
                                                          int32_t block_size, int32_t hkv, int32_t hq, int32_t vec_per_head,
                                                          int *err)
{
    // Launched as a programmatic dependent of the previous kernel in the stream (the previous
    // step's merge, whose step may still be reading the pool and the queries): wait for it before
    // any global access, then let the decode kernels launch (each of them waits for this grid
    // before it reads anything).
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
    const int64_t blk = slot / block_size, off = slot % block_size;
    const int kv_vecs = hkv * vec_per_head;
    for (int c = threadIdx.x; c < 2 * kv_vecs; c += kThreads) {
        const bool is_v = c >= kv_vecs;
        const int cc = is_v ? c - kv_vecs : c;
        const int h = cc / vec_per_head, j = cc % vec_per_head;
        const uint4 x = (is_v ? v_src : k_src)[(row * hkv + h) * vec_per_head + j];
        (is_v ? v_pool : k_pool)[((blk * hkv + h) * block_size + off) * vec_per_head + j] = x;
    }
    if (q_src) {
        const int q_vecs = hq * vec_per_head;
        const uint4 *qs = q_src + row * q_vecs;
        uint4 *qd = q_dst + i * q_vecs;
        for (int c = threadIdx.x; c < q_vecs; c += kThreads) qd[c] = qs[c];
    }
}

}  // namespace

extern "C" padoc_status padoc_append_inputs(const padoc_kv_pool *pool, const void *k_src, const void *v_src,
                                            const void *q_src, int64_t src_total, int32_t num_q_heads, void *q_dst,
                                            const int32_t *src_rows, const int32_t *slots, int32_t count,
                                            padoc_stream_t stream)
{
    if (!pool || count < 0 || src_total < 0) return PADOC_ERR_INVALID_ARGUMENT;
    if (count == 0) return PADOC_OK;
    if (!pool->k_pool || !pool->v_pool || pool->num_blocks < 1 || pool->block_size < 1 || pool->num_kv_heads < 1 ||
        pool->head_dim < 1 || !k_src || !v_src || !slots)
        return PADOC_ERR_INVALID_ARGUMENT;
    if (q_src && (!q_dst || num_q_heads < 1)) return PADOC_ERR_INVALID_ARGUMENT;
    size_t esz;
    if (pool->dtype == PADOC_DTYPE_BF16) esz = 2;
    else if (pool->dtype == PADOC_DTYPE_F32) esz = 4;
    else return PADOC_ERR_INVALID_ARGUMENT;
    const size_t row_bytes = (size_t)pool->head_dim * esz;
    if (row_bytes % 16 != 0) return PADOC_ERR_UNSUPPORTED;
    const uintptr_t align = (uintptr_t)pool->k_pool | (uintptr_t)pool->v_pool | (uintptr_t)k_src | (uintptr_t)v_src |
                            (uintptr_t)q_src | (uintptr_t)q_dst;
    if (align & 15) return PADOC_ERR_INVALID_ARGUMENT;
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
    PADOC_CUDA_TRY(cudaLaunchKernelEx(&lc, append_kernel, (const uint4 *)k_src, (const uint4 *)v_src,
                                      (const uint4 *)q_src, src_total, (uint4 *)q_dst, src_rows, slots,
                                      (uint4 *)pool->k_pool, (uint4 *)pool->v_pool,
                                      (int64_t)pool->num_blocks * pool->block_size, pool->block_size,
                                      pool->num_kv_heads, q_src ? num_q_heads : 0, (int32_t)(row_bytes / 16), err));
    return padoc_launch_status();
}
