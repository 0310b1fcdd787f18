// noalloc.cu -- the split-K decode attention for callers that cannot allocate
// device memory.
//
// loip_k_attention needs a scratch buffer for the per-page partial softmax
// states, which the caller allocates.  Some callers cannot do that: a serving
// process whose device memory is fully reserved by another allocator (for
// example a fixed arena or a caching allocator holding all of HBM), where a
// cudaMalloc would fail or break the memory budget, and latency-critical code
// that must not pay the device-wide synchronisation cudaMalloc/cudaFree imply.
// loip_k_attention_noalloc gives them the same kernel with its scratch in a
// file-scope device array, loaded with the library on every GPU that uses it
// and held until the process exits.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "../../include/loip.h"
#include "internal.h"

using namespace loip;

namespace {

// 4 Mi floats = 16 MiB of partial states, shared by every call on a device.
static __device__ __align__(256) float g_noalloc_scratch[LOIP_NOALLOC_SCRATCH_FLOATS];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
float* g_scratch_on[kMaxDevices] = {};

// Device address of the array for the current device.  In host code the
// array's name is only a host-side stand-in, so the address comes from
// cudaGetSymbolAddress, once per device, with that device current.
cudaError_t scratch_for_current_device(float** out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_scratch_on[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_on[dev] = static_cast<float*>(p);
    }
    *out = g_scratch_on[dev];
    return cudaSuccess;
}

}  // namespace

extern "C" int loip_k_attention_noalloc(const float* q, const void* kv_base, const int64_t* page_offsets,
                                        int32_t max_pages, const int32_t* ctx_lens, int32_t B, int32_t Hq, int32_t Hkv,
                                        int32_t d, int32_t page_tokens, int32_t layer, uint64_t layer_page_bytes,
                                        int32_t max_ctx, float* o, void* stream) {
    if (!q || !kv_base || !page_offsets || !ctx_lens || !o || B < 1 || Hq < 1 || Hkv < 1 || (d != 64 && d != 128) ||
        Hq % Hkv || max_ctx < 1 || page_tokens != 64 || (int64_t)max_pages * page_tokens < max_ctx)
        return LOIP_ERR_INVALID;
    // the kernel reads q and the pages with 16-byte loads, the page table as
    // int64, the lengths as int32 and writes o as fp32: a misaligned pointer is
    // refused here rather than trapping on the device
    if (((uintptr_t)q & 15) || ((uintptr_t)kv_base & 15) || ((uintptr_t)page_offsets & 7) ||
        ((uintptr_t)ctx_lens & 3) || ((uintptr_t)o & 3))
        return LOIP_ERR_INVALID;
    const int G = Hq / Hkv;  // query heads per kv head: the kernel is built for these
    if (G != 1 && G != 2 && G != 4 && G != 8) return LOIP_ERR_INVALID;
    if (attention_scratch_floats(B, Hq, d, max_ctx, page_tokens) > LOIP_NOALLOC_SCRATCH_FLOATS ||
        (max_ctx + page_tokens - 1) / page_tokens > 256)
        return LOIP_ERR_INVALID;  // the partial states and counters do not fit
    float* scratch = nullptr;
    if (scratch_for_current_device(&scratch) != cudaSuccess) return LOIP_ERR_CUDA;
    // The completion counters behind the partial states must start at zero
    // (a launch leaves them zero; clearing them here also covers the first call
    // and any earlier call that was cut short).  The partial states themselves
    // are written by the same launch before they are read.
    KvView kv{(char*)kv_base, page_offsets, max_pages, page_tokens, layer, layer_page_bytes};
    cudaError_t e = cudaMemsetAsync(attention_counters(scratch, B, Hq, d, max_ctx, page_tokens), 0,
                                    (size_t)B * Hq * sizeof(int), (cudaStream_t)stream);
    if (e != cudaSuccess) return LOIP_ERR_CUDA;
    e = launch_attention(q, kv, ctx_lens, nullptr, nullptr, B, Hq, Hkv, d, max_ctx, true, scratch, o,
                                     false, (cudaStream_t)stream);
    return e == cudaSuccess ? LOIP_OK : LOIP_ERR_CUDA;
}
