// api.cu -- status reporting, the per-device error word and tensor-map encoding for padoc_attn.
#include <cudaTypedefs.h>
#include <mutex>
#include <tuple>
#include <vector>

#include "common.cuh"

namespace {

__device__ int g_padoc_error[4];

constexpr int kMaxDevices = 64;
int *g_err_ptr[kMaxDevices] = {nullptr};
std::mutex g_mu;
thread_local int32_t t_last_code = 0, t_last_detail = 0;

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

}  // namespace

int *padoc_device_error_word()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_err_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_padoc_error) != cudaSuccess) return nullptr;
        g_err_ptr[dev] = (int *)p;
    }
    return g_err_ptr[dev];
}

namespace {

// The last few 2-D maps this thread encoded, by their arguments: a decoding loop encodes the same
// pool's maps every step, and an encoding is a pure function of its arguments.
struct TmapKey {
    int dtype;
    const void *base;
    uint64_t cols, rows, stride;
    uint32_t box_cols, box_rows;
    bool operator==(const TmapKey &o) const
    {
        return dtype == o.dtype && base == o.base && cols == o.cols && rows == o.rows && stride == o.stride &&
               box_cols == o.box_cols && box_rows == o.box_rows;
    }
};
struct TmapCache {
    TmapKey key[4];
    CUtensorMap map[4];
    bool used[4] = {false, false, false, false};
    int next = 0;
};
thread_local TmapCache t_tmaps;

bool tmap_cached(const TmapKey &k, CUtensorMap *map)
{
    for (int i = 0; i < 4; ++i)
        if (t_tmaps.used[i] && t_tmaps.key[i] == k) {
            *map = t_tmaps.map[i];
            return true;
        }
    return false;
}

void tmap_remember(const TmapKey &k, const CUtensorMap &map)
{
    const int i = t_tmaps.next;
    t_tmaps.next = (i + 1) & 3;
    t_tmaps.key[i] = k;
    t_tmaps.map[i] = map;
    t_tmaps.used[i] = true;
}

}  // namespace

padoc_status padoc_set_max_smem(const void *kernel, int bytes)
{
    // once per (kernel, size, device): the attribute stays set on the device's context
    static std::mutex mu;
    static std::vector<std::tuple<const void *, int, int>> done;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PADOC_ERR_CUDA;
    std::lock_guard<std::mutex> lk(mu);
    for (const auto &d : done)
        if (std::get<0>(d) == kernel && std::get<1>(d) == bytes && std::get<2>(d) == dev) return PADOC_OK;
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) != cudaSuccess)
        return PADOC_ERR_CUDA;
    done.emplace_back(kernel, bytes, dev);
    return PADOC_OK;
}

bool padoc_make_tmap_bf16(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows, uint64_t row_stride_bytes,
                          uint32_t box_cols, uint32_t box_rows)
{
    const TmapKey key{0, base, cols, rows, row_stride_bytes, box_cols, box_rows};
    if (tmap_cached(key, map)) return true;
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (!fn) return false;
    if ((((uintptr_t)base) & 15) || (row_stride_bytes & 15) || rows == 0 || cols == 0) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {row_stride_bytes};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return false;
    tmap_remember(key, *map);
    return true;
}

bool padoc_make_tmap_u8(CUtensorMap *map, const void *base, uint64_t cols, uint64_t rows, uint64_t row_stride_bytes,
                        uint32_t box_cols, uint32_t box_rows)
{
    const TmapKey key{1, base, cols, rows, row_stride_bytes, box_cols, box_rows};
    if (tmap_cached(key, map)) return true;
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (!fn) return false;
    if ((((uintptr_t)base) & 15) || (row_stride_bytes & 15) || rows == 0 || cols == 0 || box_cols > 128) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {row_stride_bytes};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return false;
    tmap_remember(key, *map);
    return true;
}

bool padoc_make_tmap_bf16_4d(CUtensorMap *map, const void *base, const uint64_t dims[4], const uint64_t strides_bytes[3],
                             const uint32_t box[4])
{
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (!fn) return false;
    if (((uintptr_t)base) & 15) return false;
    for (int i = 0; i < 3; ++i)
        if (strides_bytes[i] & 15) return false;
    cuuint64_t d[4] = {dims[0], dims[1], dims[2], dims[3]};
    cuuint64_t st[3] = {strides_bytes[0], strides_bytes[1], strides_bytes[2]};
    cuuint32_t bx[4] = {box[0], box[1], box[2], box[3]};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), d, st, bx, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

padoc_status padoc_launch_status()
{
    return cudaPeekAtLastError() == cudaSuccess ? PADOC_OK : (cudaGetLastError(), PADOC_ERR_CUDA);
}

int padoc_num_sms()
{
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 1;
}

extern "C" padoc_status padoc_check_device_errors(padoc_stream_t stream)
{
    t_last_code = 0;
    t_last_detail = 0;
    if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return PADOC_ERR_CUDA;
    int *p = padoc_device_error_word();
    if (!p) return PADOC_ERR_CUDA;
    int host[4] = {0, 0, 0, 0};
    if (cudaMemcpy(host, p, sizeof(host), cudaMemcpyDeviceToHost) != cudaSuccess) return PADOC_ERR_CUDA;
    if (host[0] == 0) return PADOC_OK;
    t_last_code = host[0];
    t_last_detail = host[1];
    const int zero[4] = {0, 0, 0, 0};
    if (cudaMemcpy(p, zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess) return PADOC_ERR_CUDA;
    return PADOC_ERR_DEVICE_CHECK;
}

extern "C" void padoc_last_device_error(int32_t *code, int32_t *detail)
{
    if (code) *code = t_last_code;
    if (detail) *detail = t_last_detail;
}

extern "C" const char *padoc_status_string(padoc_status status)
{
    switch (status) {
    case PADOC_OK: return "ok";
    case PADOC_ERR_INVALID_ARGUMENT: return "invalid argument";
    case PADOC_ERR_UNSUPPORTED: return "unsupported combination";
    case PADOC_ERR_WORKSPACE_TOO_SMALL: return "workspace too small";
    case PADOC_ERR_CUDA: return "CUDA error";
    case PADOC_ERR_DEVICE_CHECK: return "device-side check failed";
    case PADOC_ERR_CAPACITY: return "output capacity too small";
    }
    return "unknown status";
}

extern "C" int32_t padoc_version(void) { return PADOC_ATTN_VERSION; }
