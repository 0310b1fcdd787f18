// disktier.cpp -- the SSD tier of the weight hierarchy (HBM <- pinned host
// memory <- SSD): layers beyond the host-memory budget live in a scratch file
// and are read back with io_uring, through the raw system calls (the kernel's
// uapi header only), O_DIRECT, in 32 MB requests kept in flight together.
//
// The file is created in the caller's directory and unlinked at once, so it
// disappears with the process.  Reads complete on the ring's completion queue;
// a read's tag counts its outstanding requests.
#include "disktier.h"

#include <errno.h>
#include <fcntl.h>
#include <linux/io_uring.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include <sys/mman.h>
#include <sys/syscall.h>
#include <time.h>
#include <unistd.h>

#include <vector>

#include "../../include/loip.h"

namespace loip {

static int sys_setup(unsigned entries, io_uring_params* p) {
    return (int)syscall(__NR_io_uring_setup, entries, p);
}
static int sys_enter(int fd, unsigned to_submit, unsigned min_complete, unsigned flags) {
    return (int)syscall(__NR_io_uring_enter, fd, to_submit, min_complete, flags, nullptr, 0);
}
static uint64_t now_ms() {
    timespec ts;
    clock_gettime(CLOCK_MONOTONIC, &ts);
    return (uint64_t)ts.tv_sec * 1000ull + (uint64_t)ts.tv_nsec / 1000000ull;
}

bool DiskTier::open(const char* dir, std::string* err) {
    close();
    std::string path = std::string(dir && *dir ? dir : "/tmp") + "/loip_ssd_XXXXXX";
    std::vector<char> name(path.begin(), path.end());
    name.push_back('\0');
    int tmp = mkstemp(name.data());
    if (tmp < 0) {
        *err = std::string("cannot create the SSD-tier file in ") + (dir ? dir : "/tmp") + ": " + strerror(errno);
        return false;
    }
    ::close(tmp);
    fd_ = ::open(name.data(), O_RDWR | O_DIRECT);
    unlink(name.data());
    if (fd_ < 0) {
        *err = std::string("O_DIRECT open of the SSD-tier file failed: ") + strerror(errno);
        return false;
    }
    io_uring_params p;
    memset(&p, 0, sizeof p);
    ring_fd_ = sys_setup(64, &p);
    if (ring_fd_ < 0) {
        *err = std::string("io_uring_setup failed: ") + strerror(errno);
        close();
        return false;
    }
    entries_ = p.sq_entries;
    sq_map_ = p.sq_off.array + p.sq_entries * sizeof(unsigned);
    cq_map_ = p.cq_off.cqes + p.cq_entries * sizeof(io_uring_cqe);
    const bool single = (p.features & IORING_FEAT_SINGLE_MMAP) != 0;
    if (single) sq_map_ = cq_map_ = sq_map_ > cq_map_ ? sq_map_ : cq_map_;
    sq_ptr_ = mmap(nullptr, sq_map_, PROT_READ | PROT_WRITE, MAP_SHARED | MAP_POPULATE, ring_fd_, IORING_OFF_SQ_RING);
    if (sq_ptr_ == MAP_FAILED) sq_ptr_ = nullptr;
    cq_ptr_ = single ? sq_ptr_
                     : mmap(nullptr, cq_map_, PROT_READ | PROT_WRITE, MAP_SHARED | MAP_POPULATE, ring_fd_,
                            IORING_OFF_CQ_RING);
    if (cq_ptr_ == MAP_FAILED) cq_ptr_ = nullptr;
    sqes_map_ = p.sq_entries * sizeof(io_uring_sqe);
    sqes_ = mmap(nullptr, sqes_map_, PROT_READ | PROT_WRITE, MAP_SHARED | MAP_POPULATE, ring_fd_, IORING_OFF_SQES);
    if (sqes_ == MAP_FAILED) sqes_ = nullptr;
    if (!sq_ptr_ || !cq_ptr_ || !sqes_) {
        *err = "io_uring ring mapping failed";
        close();
        return false;
    }
    char* sq = static_cast<char*>(sq_ptr_);
    char* cq = static_cast<char*>(cq_ptr_);
    sq_head_ = reinterpret_cast<unsigned*>(sq + p.sq_off.head);
    sq_tail_ = reinterpret_cast<unsigned*>(sq + p.sq_off.tail);
    sq_mask_ = reinterpret_cast<unsigned*>(sq + p.sq_off.ring_mask);
    sq_array_ = reinterpret_cast<unsigned*>(sq + p.sq_off.array);
    cq_head_ = reinterpret_cast<unsigned*>(cq + p.cq_off.head);
    cq_tail_ = reinterpret_cast<unsigned*>(cq + p.cq_off.tail);
    cq_mask_ = reinterpret_cast<unsigned*>(cq + p.cq_off.ring_mask);
    cqes_ = cq + p.cq_off.cqes;
    in_flight_ = 0;
    for (int t = 0; t < kTags; ++t) {
        pending_[t] = 0;
        failed_[t] = false;
    }
    return true;
}

void DiskTier::close() {
    if (sqes_) munmap(sqes_, sqes_map_);
    if (cq_ptr_ && cq_ptr_ != sq_ptr_) munmap(cq_ptr_, cq_map_);
    if (sq_ptr_) munmap(sq_ptr_, sq_map_);
    sqes_ = sq_ptr_ = cq_ptr_ = nullptr;
    if (ring_fd_ >= 0) ::close(ring_fd_);
    if (fd_ >= 0) ::close(fd_);
    ring_fd_ = fd_ = -1;
}

bool DiskTier::write(uint64_t off, const void* buf, uint64_t bytes, std::string* err) {
    const char* p = static_cast<const char*>(buf);
    while (bytes) {
        const uint64_t n = bytes < (1ull << 30) ? bytes : (1ull << 30);
        ssize_t w = pwrite(fd_, p, n, (off_t)off);
        if (w <= 0) {
            *err = std::string("SSD-tier write failed: ") + (w < 0 ? strerror(errno) : "short write");
            return false;
        }
        p += w;
        off += (uint64_t)w;
        bytes -= (uint64_t)w;
    }
    return true;
}

bool DiskTier::reap(std::string* err) {
    unsigned head = __atomic_load_n(cq_head_, __ATOMIC_RELAXED);
    const unsigned tail = __atomic_load_n(cq_tail_, __ATOMIC_ACQUIRE);
    bool ok = true;
    while (head != tail) {
        const io_uring_cqe* c = static_cast<const io_uring_cqe*>(cqes_) + (head & *cq_mask_);
        const int tag = (int)(c->user_data >> 56);
        const uint64_t want = c->user_data & ((1ull << 56) - 1);
        if (tag >= 0 && tag < kTags) {
            --pending_[tag];
            if (c->res < 0 || (uint64_t)c->res != want) {
                failed_[tag] = true;
                *err = c->res < 0 ? std::string("SSD-tier read failed: ") + strerror(-c->res)
                                  : std::string("SSD-tier short read");
                ok = false;
            }
        }
        --in_flight_;
        ++head;
    }
    __atomic_store_n(cq_head_, head, __ATOMIC_RELEASE);
    return ok;
}

bool DiskTier::submit_read(uint64_t off, void* buf, uint64_t bytes, int tag, std::string* err) {
    if (tag < 0 || tag >= kTags) {
        *err = "bad read tag";
        return false;
    }
    failed_[tag] = false;
    char* p = static_cast<char*>(buf);
    while (bytes) {
        const uint64_t n = bytes < kChunk ? bytes : kChunk;
        // room in both rings: reap completions until a request fits (bounded: 60 s)
        const uint64_t deadline = now_ms() + 60000;
        while (in_flight_ >= entries_) {
            if (!reap(err)) return false;
            if (in_flight_ < entries_) break;
            if (now_ms() > deadline) {
                *err = "SSD-tier reads stopped completing";
                return false;
            }
            struct timespec ts = {0, 100000};
            nanosleep(&ts, nullptr);
        }
        const unsigned tail = __atomic_load_n(sq_tail_, __ATOMIC_RELAXED);
        const unsigned idx = tail & *sq_mask_;
        io_uring_sqe* s = static_cast<io_uring_sqe*>(sqes_) + idx;
        memset(s, 0, sizeof *s);
        s->opcode = IORING_OP_READ;
        s->fd = fd_;
        s->addr = (uint64_t)(uintptr_t)p;
        s->len = (unsigned)n;
        s->off = off;
        s->user_data = ((uint64_t)tag << 56) | n;
        sq_array_[idx] = idx;
        __atomic_store_n(sq_tail_, tail + 1, __ATOMIC_RELEASE);
        if (sys_enter(ring_fd_, 1, 0, 0) < 0) {
            *err = std::string("io_uring_enter failed: ") + strerror(errno);
            return false;
        }
        ++in_flight_;
        ++pending_[tag];
        p += n;
        off += n;
        bytes -= n;
    }
    return true;
}

bool DiskTier::wait(int tag, uint32_t timeout_ms, std::string* err) {
    const uint64_t deadline = now_ms() + timeout_ms;
    timed_out_ = false;
    while (pending_[tag] > 0) {
        if (!reap(err) && failed_[tag]) return false;
        if (pending_[tag] == 0) break;
        if (now_ms() > deadline) {
            *err = "SSD-tier read did not complete in time";
            timed_out_ = true;
            return false;
        }
        struct timespec ts = {0, 100000};  // the wait is bounded: poll the completion ring
        nanosleep(&ts, nullptr);
    }
    if (failed_[tag]) {
        if (err->empty()) *err = "SSD-tier read failed";
        return false;
    }
    return true;
}

}  // namespace loip

extern "C" int loip_ssd_roundtrip(const char* dir, uint64_t bytes, int32_t* ok) {
    using loip::DiskTier;
    if (!ok || bytes == 0 || bytes % DiskTier::kDiskAlign) return LOIP_ERR_INVALID;
    *ok = 0;
    DiskTier t;
    std::string err;
    if (!t.open(dir, &err)) return LOIP_ERR_STATE;
    void *a = nullptr, *b = nullptr;
    if (posix_memalign(&a, DiskTier::kDiskAlign, bytes) || posix_memalign(&b, DiskTier::kDiskAlign, bytes)) {
        free(a);
        return LOIP_ERR_OOM;
    }
    uint64_t* pa = static_cast<uint64_t*>(a);
    for (uint64_t i = 0; i < bytes / 8; ++i) pa[i] = i * 0x9E3779B97F4A7C15ull + 1;
    memset(b, 0, bytes);
    int rc = LOIP_OK;
    if (!t.write(0, a, bytes, &err) || !t.submit_read(0, b, bytes, 0, &err) || !t.wait(0, 60000, &err))
        rc = LOIP_ERR_STATE;
    if (rc == LOIP_OK) *ok = memcmp(a, b, bytes) == 0 ? 1 : 0;
    free(a);
    free(b);
    return rc;
}
