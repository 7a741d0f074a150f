// tc_selftest.cu -- a self-check of the tcgen05 encodings every tensor-core kernel of padoc_attn
// relies on: 128-byte-swizzled K-major and MN-major shared-memory operands, the kind::f16
// instruction descriptor, MMA completion through tcgen05.commit, and the 32x32b TMEM load layout
// (TMEM lane = accumulator row), and an A operand held in TMEM (written with tcgen05.st).
#include "common.cuh"
#include "tc.cuh"

namespace {

constexpr int kPanel = 128 * 128;   // [128 rows][64 bf16] = 16 KB
constexpr int kMat = 2 * kPanel;    // a 128 x 128 bf16 matrix as two panels
constexpr size_t kSelftestSmem = 1024 + 3 * (size_t)kMat + 64;

__global__ void __launch_bounds__(128, 1)
tc_selftest_kernel(const __nv_bfloat16 *__restrict__ a, const __nv_bfloat16 *__restrict__ bk,
                   const __nv_bfloat16 *__restrict__ v, float *__restrict__ c1, float *__restrict__ c2,
                   float *__restrict__ c3, int *err)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t *sa = smem, *sb = smem + kMat, *sv = smem + 2 * kMat;
    uint64_t *bar = (uint64_t *)(smem + 3 * kMat);
    uint32_t *tmem_slot = (uint32_t *)(bar + 1);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    // rows of 128 bf16 = 16 chunks of 16 bytes; chunk c of row r goes to panel c / 8
    for (int i = tid; i < 128 * 16; i += 128) {
        const int r = i >> 4, c = i & 15;
        const uint32_t off = (uint32_t)(c >> 3) * kPanel + sw128_offset(r, (c & 7) * 8);
        *reinterpret_cast<uint4 *>(sa + off) = *reinterpret_cast<const uint4 *>(a + r * 128 + c * 8);
        *reinterpret_cast<uint4 *>(sb + off) = *reinterpret_cast<const uint4 *>(bk + r * 128 + c * 8);
        *reinterpret_cast<uint4 *>(sv + off) = *reinterpret_cast<const uint4 *>(v + r * 128 + c * 8);
    }
    fence_proxy_async_smem();
    if (tid == 0) {
        mbar_init(smem_u32(bar), 1);
        fence_barrier_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tmem_slot), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    {   // A copied into TMEM columns 256..319: thread row r writes its 64 packed bf16 pairs
        const int row = warp * 32 + lane;
        for (int h = 0; h < 2; ++h) {
            uint32_t r[32];
            for (int j = 0; j < 32; ++j) r[j] = *reinterpret_cast<const uint32_t *>(a + row * 128 + h * 64 + 2 * j);
            tmem_st32(tmem + ((uint32_t)(warp * 32) << 16) + 256 + h * 32, r);
        }
        tmem_st_wait();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    if (tid == 0) {
        const uint32_t ua = smem_u32(sa), ub = smem_u32(sb), uv = smem_u32(sv);
        for (int ks = 0; ks < 8; ++ks) {   // C1 = A . Bk^T, both K-major
            const uint32_t off = (ks >> 2) * kPanel + (ks & 3) * 32;
            umma_bf16_ss(tmem, umma_desc_sw128(ua + off, 16, 1024), umma_desc_sw128(ub + off, 16, 1024),
                         umma_idesc_bf16(128, 128, false), ks > 0);
        }
        for (int ks = 0; ks < 8; ++ks) {   // C2 = A . V, V MN-major
            const uint32_t off = (ks >> 2) * kPanel + (ks & 3) * 32;
            umma_bf16_ss(tmem + 128, umma_desc_sw128(ua + off, 16, 1024),
                         umma_desc_sw128(uv + ks * 2048, kPanel, 1024), umma_idesc_bf16(128, 128, true), ks > 0);
        }
        for (int ks = 0; ks < 8; ++ks)     // C3 = A . V with A read from TMEM
            umma_bf16_ts(tmem + 384, tmem + 256 + ks * 8, umma_desc_sw128(uv + ks * 2048, kPanel, 1024),
                         umma_idesc_bf16(128, 128, true), ks > 0);
        umma_commit(smem_u32(bar));
    }
    __syncwarp();
    const bool ok = mbar_wait_bounded(smem_u32(bar), 0, err, 100);
    tc_fence_after();
    if (ok) {
        const int row = warp * 32 + lane;
        for (int m = 0; m < 3; ++m) {
            float *c = m == 0 ? c1 : (m == 1 ? c2 : c3);
            const int col0 = m == 2 ? 384 : m * 128;
            for (int cc = 0; cc < 4; ++cc) {
                uint32_t r[32];
                tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16) + col0 + cc * 32, r);
                tmem_ld_wait();
                for (int j = 0; j < 32; ++j) c[row * 128 + cc * 32 + j] = __uint_as_float(r[j]);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, 512);
}

// One CTA waits, with the kernels' bounded wait and a limit of limit_ns, on an mbarrier that
// nothing arrives at. Nothing else is in flight (no copy, no MMA, no tensor memory), so the CTA
// leaves cleanly once the wait gives up; every thread checks that it did give up.
__global__ void __launch_bounds__(64, 1) wait_timeout_selftest_kernel(uint64_t limit_ns, int site, int *err,
                                                                      int *gave_up)
{
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        fence_barrier_init();
    }
    __syncthreads();
    // phase 0 never completes: its one expected arrival is never made
    const bool done = mbar_wait_bounded_ns(smem_u32(&bar), 0, err, site, limit_ns);
    if (!done) atomicAdd(gave_up, 1);
}

}  // namespace

extern "C" padoc_status padoc_selftest_wait_timeout(int32_t limit_us, int32_t site, int32_t *gave_up,
                                                    padoc_stream_t stream)
{
    if (limit_us < 1 || limit_us > 100000 || site < 0 || !gave_up) return PADOC_ERR_INVALID_ARGUMENT;
    int *err = padoc_device_error_word();
    if (!err) return PADOC_ERR_CUDA;
    wait_timeout_selftest_kernel<<<1, 64, 0, (cudaStream_t)stream>>>((uint64_t)limit_us * 1000ull, site, err,
                                                                     (int *)gave_up);
    return padoc_launch_status();
}

extern "C" padoc_status padoc_selftest_tcgen05(const void *a, const void *bk, const void *v, float *c1, float *c2,
                                               float *c3, padoc_stream_t stream)
{
    if (!a || !bk || !v || !c1 || !c2 || !c3) return PADOC_ERR_INVALID_ARGUMENT;
    if ((((uintptr_t)a) | ((uintptr_t)bk) | ((uintptr_t)v)) & 15) return PADOC_ERR_INVALID_ARGUMENT;
    int *err = padoc_device_error_word();
    if (!err) return PADOC_ERR_CUDA;
    PADOC_CUDA_TRY(cudaFuncSetAttribute(tc_selftest_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSelftestSmem));
    tc_selftest_kernel<<<1, 128, kSelftestSmem, (cudaStream_t)stream>>>(
        (const __nv_bfloat16 *)a, (const __nv_bfloat16 *)bk, (const __nv_bfloat16 *)v, c1, c2, c3, err);
    return padoc_launch_status();
}
