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
//
// Huge pages: copies out of base (64 KB) pages ran 3-15x slower than out of
// huge pages (12-80 GB/s against 211), and a buffer allocated while host memory
// is fragmented (right after another process freed a large pool) can come back
// partly in base pages.  So every buffer spans whole huge pages, is collapsed
// into huge pages after its first touch (MADV_COLLAPSE, where the kernel has
// it), and reports the share of it that /proc/self/smaps shows as huge pages;
// the runtime re-allocates buffers that are not entirely huge.
//
// Placement: before the first touch the mapping is given the memory policy
// MPOL_PREFERRED for the host NUMA node closest to the GPU
// (cudaDevAttrHostNumaId), so that its pages come from the memory next to the
// link the copy engine reads over (preferred, not bound: when that node runs
// out the kernel falls back to another node instead of failing the fault).  The
// runtime reads back where the pages landed (move_pages queries).
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include <sys/mman.h>
#include <sys/stat.h>
#include <sys/syscall.h>
#include <unistd.h>

#include <vector>

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

int gpu_host_node() {
    int dev = 0, node = -1;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&node, cudaDevAttrHostNumaId, dev) != cudaSuccess) {
        cudaGetLastError();
        return -1;
    }
    if (node < 0 || node >= 1024) return -1;
    char path[64];
    snprintf(path, sizeof path, "/sys/devices/system/node/node%d", node);
    struct stat st;
    return stat(path, &st) == 0 ? node : -1;
}

// MPOL_PREFERRED for `node` on [p, p + bytes) (Linux memory-policy constant).
static bool prefer_node(void* p, size_t bytes, int node) {
    constexpr int kMpolPreferred = 1;
    unsigned long mask[1024 / (8 * sizeof(unsigned long))] = {};
    mask[node / (8 * sizeof(unsigned long))] |= 1ul << (node % (8 * sizeof(unsigned long)));
    return syscall(SYS_mbind, p, bytes, kMpolPreferred, mask, (unsigned long)1024, 0u) == 0;
}

// Share of [p, p + span) (one VMA of its own) that smaps counts as AnonHugePages.
static double huge_fraction(const void* p, size_t span) {
    FILE* f = fopen("/proc/self/smaps", "r");
    if (!f) return 0.0;
    const uintptr_t a = reinterpret_cast<uintptr_t>(p);
    char line[512];
    bool in = false;
    double frac = 0.0;
    while (fgets(line, sizeof line, f)) {
        unsigned long lo = 0, hi = 0;
        if (sscanf(line, "%lx-%lx ", &lo, &hi) == 2 && strchr(line, '-') < strchr(line, ' ')) {
            if (in) break;
            in = a >= lo && a < hi;
            continue;
        }
        unsigned long kb = 0;
        if (in && sscanf(line, "AnonHugePages: %lu kB", &kb) == 1) {
            frac = (double)kb * 1024.0 / (double)span;
            break;
        }
    }
    fclose(f);
    return frac > 1.0 ? 1.0 : frac;
}

int host_range_node(const void* p, size_t bytes, int samples, double* frac) {
    if (frac) *frac = 0.0;
    if (!p || bytes == 0 || samples < 1) return -1;
    const size_t pg = (size_t)sysconf(_SC_PAGESIZE);
    std::vector<void*> pages(samples);
    std::vector<int> status(samples, -1);
    for (int i = 0; i < samples; ++i) {
        const uintptr_t a = reinterpret_cast<uintptr_t>(p) + (bytes - 1) * (size_t)i / (size_t)(samples > 1 ? samples - 1 : 1);
        pages[i] = reinterpret_cast<void*>(a / pg * pg);
    }
    if (syscall(SYS_move_pages, 0, (unsigned long)samples, pages.data(), nullptr, status.data(), 0) != 0) return -1;
    int best = -1, best_n = 0;
    for (int i = 0; i < samples; ++i) {
        if (status[i] < 0) continue;
        int n = 0;
        for (int j = 0; j < samples; ++j) n += status[j] == status[i];
        if (n > best_n) {
            best_n = n;
            best = status[i];
        }
    }
    if (frac) *frac = (double)best_n / samples;
    return best;
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
    // whole huge pages: the buffer is rounded up to the huge-page size, so its
    // last part is a huge page too (a partial one falls back to base pages,
    // and copies out of them ran 3-8x slower)
    const size_t span = (bytes + hp - 1) / hp * hp;
    const size_t map_bytes = span + hp;
    void* base = mmap(nullptr, map_bytes, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
    if (base != MAP_FAILED) {
        char* p = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(base) + hp - 1) / hp * hp);
        const int node = gpu_host_node();
        const bool placed = node >= 0 && prefer_node(p, span, node);
        madvise(p, span, MADV_HUGEPAGE);
        memset(p, 0, span);
        constexpr int kMadvCollapse = 25;  // Linux MADV_COLLAPSE (6.1+); EINVAL elsewhere, ignored
        madvise(p, span, kMadvCollapse);
        const double huge = huge_fraction(p, span);
        if (cudaHostRegister(p, span, cudaHostRegisterPortable | cudaHostRegisterMapped) == cudaSuccess) {
            out->base = base;
            out->map_bytes = map_bytes;
            out->ptr = p;
            out->bytes = bytes;
            out->mapped = true;
            out->node = placed ? node : -1;
            out->huge = huge;
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
