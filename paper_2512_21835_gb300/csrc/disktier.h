// disktier.h -- the SSD tier: layer blobs in a file, read with io_uring (see disktier.cpp).
#pragma once
#include <stdint.h>

#include <string>

namespace loip {

// One unlinked scratch file in `dir` (opened O_DIRECT) plus an io_uring instance
// driven through the raw system calls.  Offsets, sizes and buffers of reads and
// writes must be multiples of kDiskAlign.  Not thread-safe; one per context.
class DiskTier {
   public:
    static constexpr uint64_t kDiskAlign = 4096;
    static constexpr uint64_t kChunk = 32ull << 20;  // bytes per read request

    ~DiskTier() { close(); }
    // false (and *err set) if the file or the ring cannot be created
    bool open(const char* dir, std::string* err);
    void close();
    bool is_open() const { return fd_ >= 0; }
    // synchronous write of `bytes` at `off`
    bool write(uint64_t off, const void* buf, uint64_t bytes, std::string* err);
    // queues reads of [off, off + bytes) into buf (kChunk per request) under `tag`
    bool submit_read(uint64_t off, void* buf, uint64_t bytes, int tag, std::string* err);
    // waits until every read queued under `tag` has completed; false on an I/O
    // error or when timeout_ms passes (then *err says which)
    bool wait(int tag, uint32_t timeout_ms, std::string* err);
    // whether the last failed wait() ran out of time (else it saw an I/O error)
    bool timed_out() const { return timed_out_; }

   private:
    bool reap(std::string* err);  // drains the completion ring
    int fd_ = -1, ring_fd_ = -1;
    void* sq_ptr_ = nullptr;
    void* cq_ptr_ = nullptr;
    void* sqes_ = nullptr;
    uint64_t sq_map_ = 0, cq_map_ = 0, sqes_map_ = 0;
    unsigned *sq_head_ = nullptr, *sq_tail_ = nullptr, *sq_mask_ = nullptr, *sq_array_ = nullptr;
    unsigned *cq_head_ = nullptr, *cq_tail_ = nullptr, *cq_mask_ = nullptr;
    void* cqes_ = nullptr;
    unsigned entries_ = 0, in_flight_ = 0;
    static constexpr int kTags = 8;
    int pending_[kTags] = {};
    bool failed_[kTags] = {};
    bool timed_out_ = false;
};

}  // namespace loip
