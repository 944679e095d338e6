// libsonic: status reporting and host helpers shared by the entry points.
#include <cudaTypedefs.h>

#include <mutex>

#include "sonic_host.h"

namespace sonic {

namespace {
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}
}  // namespace

bool make_tmap_bf16_4d(CUtensorMap *map, const void *base, const uint64_t dims[4],
                       const uint64_t strides[3], const uint32_t box[4]) {
    auto fn = encode_fn();
    if (fn == nullptr) return false;
    cuuint64_t gdim[4] = {dims[0], dims[1], dims[2], dims[3]};
    cuuint64_t gstride[3] = {strides[0], strides[1], strides[2]};
    cuuint32_t bdim[4] = {box[0], box[1], box[2], box[3]};
    cuuint32_t estride[4] = {1, 1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), gdim,
                    gstride, bdim, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_tmap_bf16_5d(CUtensorMap *map, const void *base, const uint64_t dims[5],
                       const uint64_t strides[4], const uint32_t box[5]) {
    auto fn = encode_fn();
    if (fn == nullptr) return false;
    cuuint64_t gdim[5] = {dims[0], dims[1], dims[2], dims[3], dims[4]};
    cuuint64_t gstride[4] = {strides[0], strides[1], strides[2], strides[3]};
    cuuint32_t bdim[5] = {box[0], box[1], box[2], box[3], box[4]};
    cuuint32_t estride[5] = {1, 1, 1, 1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void *>(base), gdim,
                    gstride, bdim, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

int device_sm_count() {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    if (dev >= 0 && dev < 64 && cache[dev] > 0) return cache[dev];
    int n = 1;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (dev >= 0 && dev < 64) cache[dev] = n;
    return n;
}

}  // namespace sonic

extern "C" sonic_status_t sonic_read_status(const int32_t *status, sonic_stream_t stream) {
    if (status == nullptr) return SONIC_ERR_INVALID_ARGUMENT;
    int32_t h = 0;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(&h, status, sizeof(h), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return SONIC_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return SONIC_ERR_CUDA;
    return static_cast<sonic_status_t>(h);
}

extern "C" const char *sonic_status_string(sonic_status_t st) {
    switch (st) {
        case SONIC_OK: return "ok";
        case SONIC_ERR_INVALID_ARGUMENT: return "invalid argument";
        case SONIC_ERR_UNSUPPORTED: return "unsupported configuration";
        case SONIC_ERR_WORKSPACE: return "workspace missing or too small";
        case SONIC_ERR_CAPACITY: return "output capacity exceeded";
        case SONIC_ERR_DEVICE_TIMEOUT: return "device wait timed out";
        case SONIC_ERR_CUDA: return "CUDA error";
        case SONIC_ERR_LAYOUT: return "inconsistent role/segment layout";
    }
    return "unknown status";
}

extern "C" int32_t sonic_abi_version(void) { return SONIC_ABI_VERSION; }
