// hostpool.cpp -- pinned host memory for the offloaded-layer pool.
//
// The copy engine reads the pool over the host link once per offloaded layer
// and step, so how the pool's physical pages are laid out matters.  Measured
// on the GB300 host (64 KB base pages, 512 MB transparent huge pages), copying
// 50 layer blobs of 1.71 GB into two device slots:
//   cudaHostAlloc per blob                                193-211 GB/s
//   huge-page region registered untouched                 181-212 GB/s
//   huge-page region per blob, registered untouched        84-192 GB/s
//   huge-page region, written once, then registered       211-212 GB/s
// so a buffer is an anonymous mapping aligned to the huge-page size, advised
// MADV_HUGEPAGE, written through once in address order (which also faults its
// pages in), then registered with cudaHostRegister; cudaHostAlloc is the
// fallback when that fails.  Every buffer is registered mapped, so kernels can
// also read it in place through its device address (direct-access decode).
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include <sys/mman.h>
#include <unistd.h>

#include "hostpool.h"

namespace loip {

static size_t huge_page_bytes() {
    static size_t hp = 0;
    if (hp) return hp;
    hp = 2u << 20;
    FILE* f = fopen("/sys/kernel/mm/transparent_hugepage/hpage_pmd_size", "r");
    if (f) {
        unsigned long long v = 0;
        if (fscanf(f, "%llu", &v) == 1 && v >= 4096 && v <= (1ull << 31)) hp = (size_t)v;
        fclose(f);
    }
    return hp;
}

// Device address of the buffer on the current device (nullptr when the driver
// cannot map it; direct-access users check for that).
static void map_device(HostBuf* b) {
    void* d = nullptr;
    if (cudaHostGetDevicePointer(&d, b->ptr, 0) == cudaSuccess) {
        b->dev = d;
    } else {
        cudaGetLastError();
        b->dev = nullptr;
    }
}

cudaError_t host_buf_alloc(size_t bytes, HostBuf* out) {
    *out = HostBuf{};
    if (bytes == 0) return cudaSuccess;
    // LOIP_HOST_POOL=hostalloc selects plain cudaHostAlloc (kept for measuring the two side by side)
    static const char* mode = getenv("LOIP_HOST_POOL");
    if (mode && strcmp(mode, "hostalloc") == 0) {
        void* q = nullptr;
        cudaError_t e = cudaHostAlloc(&q, bytes, cudaHostAllocPortable | cudaHostAllocMapped);
        if (e != cudaSuccess) return e;
        out->ptr = q;
        out->bytes = bytes;
        map_device(out);
        return cudaSuccess;
    }
    const size_t hp = huge_page_bytes();
    const size_t map_bytes = bytes + hp;
    void* base = mmap(nullptr, map_bytes, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
    if (base != MAP_FAILED) {
        char* p = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(base) + hp - 1) / hp * hp);
        madvise(p, bytes, MADV_HUGEPAGE);
        memset(p, 0, bytes);
        if (cudaHostRegister(p, bytes, cudaHostRegisterPortable | cudaHostRegisterMapped) == cudaSuccess) {
            out->base = base;
            out->map_bytes = map_bytes;
            out->ptr = p;
            out->bytes = bytes;
            out->mapped = true;
            map_device(out);
            return cudaSuccess;
        }
        cudaGetLastError();  // clear the failed registration
        munmap(base, map_bytes);
    }
    void* q = nullptr;
    cudaError_t e = cudaHostAlloc(&q, bytes, cudaHostAllocPortable | cudaHostAllocMapped);
    if (e != cudaSuccess) return e;
    out->ptr = q;
    out->bytes = bytes;
    out->mapped = false;
    map_device(out);
    return cudaSuccess;
}

cudaError_t host_buf_alloc_plain(size_t bytes, HostBuf* out) {
    *out = HostBuf{};
    if (bytes == 0) return cudaSuccess;
    void* q = nullptr;
    cudaError_t e = cudaHostAlloc(&q, bytes, cudaHostAllocPortable | cudaHostAllocMapped);
    if (e != cudaSuccess) return e;
    out->ptr = q;
    out->bytes = bytes;
    out->mapped = false;
    map_device(out);
    return cudaSuccess;
}

void host_buf_free(HostBuf* b) {
    if (!b->ptr) return;
    if (b->mapped) {
        cudaHostUnregister(b->ptr);
        munmap(b->base, b->map_bytes);
    } else {
        cudaFreeHost(b->ptr);
    }
    *b = HostBuf{};
}

}  // namespace loip
