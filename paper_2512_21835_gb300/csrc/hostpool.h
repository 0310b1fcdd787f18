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
// plain cudaHostAlloc buffer (the SSD tier's staging buffers: O_DIRECT reads
// land in them, and copies out of registered huge-page mappings that direct I/O
// keeps rewriting ran at ~3 GB/s against the disk's 9 GB/s)
cudaError_t host_buf_alloc_plain(size_t bytes, HostBuf* out);
void host_buf_free(HostBuf* b);
}  // namespace loip
