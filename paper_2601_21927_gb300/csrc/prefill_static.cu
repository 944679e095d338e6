// sonic_attn_prefill_static: the masked prefill for callers that cannot
// allocate device memory.
//
// Some callers cannot call cudaMalloc at all: code running inside a custom
// allocator or a memory-pool callback, runtimes that pre-plan every byte of
// device memory up front, or hosts that only hand out fixed buffers for the
// model's tensors.  They can still pass inputs and outputs, but not the
// caller-owned workspace sonic_attn_prefill needs for its per-tile mask
// summaries.  This entry point keeps that scratch in a fixed array compiled
// into the library instead, and runs the same kernels.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds it until the process exits.  In host code its name is only a
// host-side stand-in, so its device address is looked up with
// cudaGetSymbolAddress once per device (with that device current) on the
// first call made on that device, and cached together with the unique id of
// the context it belongs to.  A device reset destroys that context and the
// module loaded into it; the next call sees a different context id and looks
// the address up again instead of handing the kernels a dead address.
#include <cudaTypedefs.h>

#include <mutex>

#include "sonic_host.h"

namespace {

// 9 MiB + 256 bytes: the work-unit counter and room for 32768 key tiles, each
// with a 32-byte summary and a 256-byte column-mask record, i.e.
// batch * ceil(max_k_len / 128) <= 32768 (for example 64 sequences of up to
// 65536 keys).
constexpr size_t kStaticScratchBytes = (size_t(9) << 20) + 256;

static __device__ __align__(256) unsigned char g_prefill_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
void *g_scratch_ptr[kMaxDevices] = {nullptr};
unsigned long long g_scratch_ctx[kMaxDevices] = {0};
std::mutex g_scratch_mu;

// Unique id of the calling thread's current context (0 when there is none or
// the driver cannot say).  Ids are never reused within a process.
unsigned long long current_context_id() {
    static PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
    static PFN_cuCtxGetId_v12000 get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(p);
    });
    if (get_current == nullptr || get_id == nullptr) return 0;
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
    if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of the scratch array on the current device: looked up once
// per device and context, then served from the cache.
sonic_status_t scratch_address(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return SONIC_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return SONIC_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    const unsigned long long ctx = current_context_id();
    if (g_scratch_ptr[dev] == nullptr || ctx == 0 || ctx != g_scratch_ctx[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_prefill_scratch) != cudaSuccess || p == nullptr)
            return SONIC_ERR_CUDA;
        g_scratch_ptr[dev] = p;
        // the lookup made the device's primary context current if it was not
        g_scratch_ctx[dev] = current_context_id();
    }
    *out = g_scratch_ptr[dev];
    return SONIC_OK;
}

}  // namespace

extern "C" sonic_status_t sonic_attn_prefill_static(const uint16_t *Q, const uint16_t *K,
                                                    const uint16_t *V, const int32_t *seg_id,
                                                    const uint8_t *role, uint16_t *O,
                                                    const sonic_prefill_args *args,
                                                    sonic_stream_t stream) {
    if (args == nullptr) return SONIC_ERR_INVALID_ARGUMENT;
    // the retained-first order copies K and V into the workspace: not here
    if (args->key_order != SONIC_KEYS_AS_GIVEN) return SONIC_ERR_UNSUPPORTED;
    sonic_prefill_args a = *args;
    a.workspace = nullptr;
    a.workspace_bytes = 0;
    const size_t need = sonic_prefill_workspace_size(&a);
    if (need > kStaticScratchBytes) return SONIC_ERR_WORKSPACE;
    if (need > 0) {
        void *p = nullptr;
        const sonic_status_t st = scratch_address(&p);
        if (st != SONIC_OK) return st;
        a.workspace = p;
        a.workspace_bytes = kStaticScratchBytes;
    }
    return sonic_attn_prefill(Q, K, V, seg_id, role, O, &a, stream);
}
