// common.cuh -- device helpers of padoc_attn (sm_103a): error word, bounded mbarrier waits,
// TMA tile loads, warp-level bf16 MMA, and host helpers for tensor maps and launches.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "padoc_attn.h"
#include "plan_internal.h"

// ------------------------------------------------------------------------------------------------
// Device error word: [0] = code (first error wins), [1] = detail.
// ------------------------------------------------------------------------------------------------
#define PADOC_DEVERR_BLOCK_ID 1
#define PADOC_DEVERR_TIMEOUT 2
#define PADOC_DEVERR_SMEM_ALIGN 3

__device__ __forceinline__ void padoc_record_error(int *err, int code, int detail)
{
    if (atomicCAS(err, 0, code) == 0) atomicExch(err + 1, detail);
}

// Upper bound of any single wait inside a kernel (ns of %globaltimer).
#define PADOC_WAIT_LIMIT_NS 2000000000ull

__device__ __forceinline__ uint64_t padoc_globaltimer()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ------------------------------------------------------------------------------------------------
// mbarrier
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_barrier_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n"
        " mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Waits for the phase with the given parity to complete; false (and the error word set to
// PADOC_DEVERR_TIMEOUT with `site` as the detail) if it does not complete within limit_ns.
__device__ __forceinline__ bool mbar_wait_bounded_ns(uint32_t bar, uint32_t parity, int *err, int site,
                                                     uint64_t limit_ns)
{
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = padoc_globaltimer();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 255u) == 0 && padoc_globaltimer() - t0 > limit_ns) {
            padoc_record_error(err, PADOC_DEVERR_TIMEOUT, site);
            return false;
        }
    }
}

// The kernels' wait: mbar_wait_bounded_ns with the library's limit, PADOC_WAIT_LIMIT_NS.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, int *err, int site)
{
    return mbar_wait_bounded_ns(bar, parity, err, site, PADOC_WAIT_LIMIT_NS);
}

// ------------------------------------------------------------------------------------------------
// TMA (cp.async.bulk.tensor), 2-D tiles into shared memory, completion on an mbarrier.
// x is the innermost coordinate (elements); callers keep x * sizeof(elem) a multiple of 16.
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int32_t x, int32_t y, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// L2 policy for data read once per call (the paged K/V): such lines are the first evicted, so the
// split-K partials written in the same call stay in L2 for the merge that reads them.
__device__ __forceinline__ uint64_t l2_evict_first_policy()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

__device__ __forceinline__ uint64_t l2_evict_normal_policy()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// tma_load_2d with an L2 cache policy.
__device__ __forceinline__ void tma_load_2d_hint(uint32_t dst, const CUtensorMap *map, int32_t x, int32_t y, uint32_t bar,
                                                 uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(policy)
        : "memory");
}

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *map, int32_t c0, int32_t c1, int32_t c2,
                                            int32_t c3, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
        : "memory");
}

// Contiguous bulk copy global -> shared (both addresses 16-byte aligned, bytes a multiple of 16),
// completion on an mbarrier.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

// Pulls a 2-D box into L2 without a destination or completion signal (out-of-range parts fetch nothing).
__device__ __forceinline__ void tma_prefetch_l2_2d(const CUtensorMap *map, int32_t c0, int32_t c1)
{
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(reinterpret_cast<uint64_t>(map)),
                 "r"(c0), "r"(c1)
                 : "memory");
}

// Pulls a 4-D box into L2 without a destination or completion signal.
__device__ __forceinline__ void tma_prefetch_l2_4d(const CUtensorMap *map, int32_t c0, int32_t c1, int32_t c2, int32_t c3)
{
    asm volatile("cp.async.bulk.prefetch.tensor.4d.L2.global.tile [%0, {%1, %2, %3, %4}];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(c0), "r"(c1), "r"(c2), "r"(c3)
                 : "memory");
}

__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap *map)
{
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ------------------------------------------------------------------------------------------------
// cp.async (16 bytes per thread, L2 only). A source size of 0 fills the 16 bytes with zeros.
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ void cp_async_16(uint32_t dst, const void *src, uint32_t src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
// cp_async_16 with an L2 cache policy.
__device__ __forceinline__ void cp_async_16_hint(uint32_t dst, const void *src, uint32_t src_bytes, uint64_t policy)
{
    asm volatile("cp.async.cg.shared.global.L2::cache_hint [%0], [%1], 16, %2, %3;" ::"r"(dst), "l"(src), "r"(src_bytes),
                 "l"(policy)
                 : "memory");
}
// 4 bytes through L1 (cp.async of fewer than 16 bytes takes the .ca form); src_bytes 0 writes zeros.
__device__ __forceinline__ void cp_async_4(uint32_t dst, const void *src, uint32_t src_bytes)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }
// Arrives on the mbarrier once every cp.async this thread issued so far has completed; the arrival is
// one of the barrier's expected arrivals (no pending-count increment).
__device__ __forceinline__ void cp_async_mbar_arrive(uint32_t bar)
{
    asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}

// Byte offset of element (row, col) of a [rows][64] bf16 panel written by TMA with 128-byte
// swizzle (16-byte chunk index XOR row % 8); panels start on 1024-byte boundaries.
__device__ __forceinline__ uint32_t sw128_offset(uint32_t row, uint32_t col)
{
    return row * 128u + ((((col >> 3) ^ row) & 7u) << 4) + ((col & 7u) << 1);
}

// ------------------------------------------------------------------------------------------------
// Warp-level MMA (mma.sync m16n8k16 bf16 -> fp32), ldmatrix, movmatrix
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t (&r)[4], uint32_t addr)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t x)
{
    uint32_t y;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

__device__ __forceinline__ float fast_exp2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// ------------------------------------------------------------------------------------------------
// E4M3 (the OCP 8-bit floating point format, 4 exponent bits with bias 7, 3 mantissa bits, no
// infinities, largest finite 448) conversions of the FP8 KV cache.
// ------------------------------------------------------------------------------------------------
// Two codes (low byte first) to an f16x2: exact (every E4M3 value is an f16 normal or zero).
__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint16_t c)
{
    uint32_t h;
    asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(h) : "h"(c));
    return h;
}

// Two codes to a bf16x2 holding code_value * 2^-112, exactly: the f16 bits with the exponent and
// the top 7 mantissa bits moved down three places (E4M3 values use only the top 3 of f16's 10
// mantissa bits) read as bf16 with exponent field 0..23 instead of f16's biased exponent, i.e.
// the value times 2^(15 - 127); every nonzero result is a bf16 normal (no subnormal operand
// reaches the tensor cores). Callers fold 2^112 into the scale they apply.
#define PADOC_E4M3_BF16_SHIFT_LOG2 112
__device__ __forceinline__ uint32_t e4m3x2_to_bf16x2_shifted(uint16_t c)
{
    const uint32_t h = e4m3x2_to_f16x2(c);
    const uint32_t mag = (h & 0x7FFF7FFFu) >> 3;   // the high half's low mantissa bits are zero
    return mag | (h & 0x80008000u);
}

// The exact fp32 value of one code.
__device__ __forceinline__ float e4m3_to_f32(uint8_t c)
{
    const uint32_t h = e4m3x2_to_f16x2((uint16_t)c);
    return __half2float(__ushort_as_half((unsigned short)(h & 0xFFFFu)));
}

// Codes of two fp32 values (lo -> low byte), nearest even, magnitudes past 448 saturated to 448.
__device__ __forceinline__ uint16_t f32x2_to_e4m3x2(float lo, float hi)
{
    uint16_t c;
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(c) : "f"(hi), "f"(lo));
    return c;
}

// Programmatic dependent launch: a grid lets the next grid in its stream start launching, and a
// dependent grid waits until its prerequisite grid has completed and its writes are visible.
// One 32-byte store of eight floats (p 32-byte aligned): a whole sector per lane.
__device__ __forceinline__ void st_global_v8(float *p, float a0, float a1, float a2, float a3, float a4, float a5,
                                             float a6, float a7)
{
    asm volatile("st.global.v8.f32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "f"(a0), "f"(a1), "f"(a2),
                 "f"(a3), "f"(a4), "f"(a5), "f"(a6), "f"(a7)
                 : "memory");
}

// Named barrier `id` (1..15) over `count` threads (a multiple of 32) of the CTA.
__device__ __forceinline__ void named_bar_sync(int id, int count)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Per-thread register budget of the executing warpgroup (all four warps run the same instruction):
// inc waits until the CTA's pool (what its threads were launched with) has the registers; dec
// returns registers to it. N is a multiple of 8 in [24, 256].
template <uint32_t N>
__device__ __forceinline__ void setmaxnreg_inc()
{
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(N));
}
template <uint32_t N>
__device__ __forceinline__ void setmaxnreg_dec()
{
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(N));
}
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait_prerequisite() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

#define PADOC_LOG2E 1.4426950408889634f
#define PADOC_LN2 0.6931471805599453f

// ------------------------------------------------------------------------------------------------
// Host helpers (defined in api.cu)
// ------------------------------------------------------------------------------------------------
// Device address of the current device's error word (set up once per device).
int *padoc_device_error_word();
// 2-D bf16 tensor map: rows x cols elements with a row pitch of `row_stride_bytes`, box of
// box_rows x 64 columns, 128-byte swizzle. Returns false if the driver rejects it.
// cudaFuncSetAttribute(kernel, MaxDynamicSharedMemorySize, bytes), once per kernel, size and device.
padoc_status padoc_set_max_smem(const void *kernel, int bytes);
bool padoc_make_tmap_bf16(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows,
                          uint64_t row_stride_bytes, uint32_t box_cols, uint32_t box_rows);
// 2-D uint8 tensor map (E4M3 codes): rows x cols bytes with a row pitch of `row_stride_bytes`, box of
// box_rows x box_cols bytes (box_cols <= 128), 128-byte swizzle.
bool padoc_make_tmap_u8(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows, uint64_t row_stride_bytes,
                        uint32_t box_cols, uint32_t box_rows);
// 4-D bf16 tensor map (dims[0] innermost, strides of dims 1..3 in bytes), 128-byte swizzle.
bool padoc_make_tmap_bf16_4d(CUtensorMap *map, const void *base, const uint64_t dims[4], const uint64_t strides_bytes[3],
                             const uint32_t box[4]);
padoc_status padoc_launch_status();
// tcgen05 packed prefill (prefill_tc.cu); arguments validated by the caller.
padoc_status padoc_launch_prefill_tc(const void *q, const void *k, const void *v, int64_t total_tokens,
                                     int32_t num_q_heads, int32_t num_kv_heads, const int32_t *spans_dev,
                                     const int32_t *tile_row_ptr_dev, const int32_t *tile_k_dev,
                                     const int8_t *tile_kind_dev, float scale_log2, void *out, float *lse,
                                     cudaStream_t stream);
namespace padoc_warp {
struct DecodeParams;
}
// The decode grid (decode_tc.cu): the plan's tensor-core items, then its warp lists (wprm, the
// warp path's arguments). k_scales / v_scales non-null: an E4M3 pool (kmap / vmap are
// padoc_make_tmap_u8 maps of the codes), whose grid runs the tensor-core items only (the caller
// launches decode_warp_kernel after it).
padoc_status padoc_launch_decode_tc(const CUtensorMap *kmap, const CUtensorMap *vmap, const CUtensorMap *qmap, const int32_t *plan,
                                    const padoc_decode_plan *info, const int32_t *page_table, int32_t page_stride,
                                    const int32_t *stream_table, int32_t stream_stride, int32_t num_blocks,
                                    const float *k_scales, const float *v_scales, __nv_bfloat16 *part_o, float *part_lse,
                                    __nv_bfloat16 *out, float *lse, float scale_log2, int *err,
                                    const padoc_warp::DecodeParams *wprm, cudaStream_t stream);
// tcgen05 prefill backward (prefill_bwd_tc.cu): the dQ pass, which also writes lt / dt (per head
// [Hq][t_pad]: -lse2 and rowsum(dO * O)), then the dK/dV pass; arguments validated by the caller.
padoc_status padoc_launch_prefill_bwd_tc(const void *q, const void *k, const void *v, const void *out,
                                         const void *dout, const float *lse, int64_t total_tokens,
                                         int32_t num_q_heads, int32_t num_kv_heads, const int32_t *spans_dev,
                                         const padoc_tile_map_dev *q_map, const padoc_tile_map_dev *k_map, float *lt,
                                         float *dt, float *split, int64_t t_pad, float scale, void *dq, void *dk,
                                         void *dv, cudaStream_t stream);
int padoc_num_sms();
// SM count the planner sizes grids for (the current device's, read once; 152 without a device)
int32_t padoc_default_ctas();

#define PADOC_CUDA_TRY(expr)                                   \
    do {                                                       \
        if ((expr) != cudaSuccess) return PADOC_ERR_CUDA;      \
    } while (0)
