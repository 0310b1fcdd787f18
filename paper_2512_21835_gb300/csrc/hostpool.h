// hostpool.h -- pinned, huge-page-backed host buffers (see hostpool.cpp).
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>

namespace loip {
struct HostBuf {
    void* base = nullptr;  // mapping start (mapped buffers)
    size_t map_bytes = 0;
    void* ptr = nullptr;   // usable, registered pointer
    size_t bytes = 0;
    bool mapped = false;   // mmap + cudaHostRegister (else cudaHostAlloc)
    void* dev = nullptr;   // device address of ptr (registered mapped), or nullptr
};
cudaError_t host_buf_alloc(size_t bytes, HostBuf* out);
void host_buf_free(HostBuf* b);
}  // namespace loip
