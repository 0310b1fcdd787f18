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
    int node = -1;         // host NUMA node the pages were asked for (-1: none)
    double huge = 0.0;     // share of the buffer in transparent huge pages (1 = all)
};
// Host NUMA node closest to the current device (cudaDevAttrHostNumaId), or -1
// when the system reports none or the node does not exist on this host.
int gpu_host_node();
// Majority NUMA node of `samples` pages spread evenly over [p, p + bytes)
// (move_pages query, pages already touched); *frac gets the share of sampled
// pages on that node.  -1 when the kernel cannot tell.
int host_range_node(const void* p, size_t bytes, int samples, double* frac);
cudaError_t host_buf_alloc(size_t bytes, HostBuf* out);
// plain cudaHostAlloc buffer (the SSD tier's staging buffers: O_DIRECT reads
// land in them, and copies out of registered huge-page mappings that direct I/O
// keeps rewriting ran at ~3 GB/s against the disk's 9 GB/s)
cudaError_t host_buf_alloc_plain(size_t bytes, HostBuf* out);
void host_buf_free(HostBuf* b);
}  // namespace loip
