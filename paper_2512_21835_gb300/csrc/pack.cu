// pack.cu -- lossless packing of bf16 weights for the host link.
//
// The streamed layers cross the host link every step, and the link is the
// step's bound, so the stream carries fewer bytes without changing a single
// weight: each bf16 word w = [sign | exponent (8) | mantissa (7)] is split into
// its sign-and-mantissa byte, stored as is, and its exponent, stored as a 4-bit
// code relative to the largest exponent of its superblock (1024 words).  Model
// weights of one superblock span far fewer than 2^8 binades, so nearly every
// exponent lies within the 15 binades below that maximum; the rest are kept as
// exceptions.  Decoding restores every word bit for bit.
//
// Packed superblock (kPackedSb = 1568 bytes for 1024 words = 2048 bytes):
//   bytes    0 .. 1023  sign-and-mantissa byte of word i: (w >> 8 & 0x80) | (w & 0x7f)
//   bytes 1024 .. 1535  4-bit codes, word i in byte 1024 + i / 2 (low nibble for even i):
//                       code c in 1..15: exponent = base + c - 15; code 0: an exception
//   bytes 1536 .. 1567  record: byte 0 base (the largest exponent), byte 1 the number
//                       of exceptions (0..7, or 0xff: the superblock is not packed --
//                       more than 7 exceptions -- and its 2048 raw bytes travel
//                       separately), bytes 4 + 4k: exception k = index | exponent << 16
//
// One warp per superblock in both directions; lane j handles words 32 j .. 32 j + 31.
#include <cuda_runtime.h>
#include <stdint.h>

#include "internal.h"

namespace loip {
namespace {

constexpr int kWarps = 8;  // superblocks per 256-thread block

__global__ void __launch_bounds__(256) pack_kernel(const uint16_t* __restrict__ in, uint64_t n_sb,
                                                   uint8_t* __restrict__ out, uint32_t* raw_list, uint32_t first_sb,
                                                   uint32_t raw_cap) {
    const uint64_t sb = (uint64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
    if (sb >= n_sb) return;
    const int lane = threadIdx.x & 31;
    const uint4* src = reinterpret_cast<const uint4*>(in + sb * kPackWords + lane * 32);
    uint32_t w[16];  // 32 words, two per register
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint4 v = src[i];
        w[4 * i] = v.x;
        w[4 * i + 1] = v.y;
        w[4 * i + 2] = v.z;
        w[4 * i + 3] = v.w;
    }
    auto word = [&](int i) -> uint32_t { return (w[i >> 1] >> ((i & 1) * 16)) & 0xffffu; };
    uint32_t emax = 0;
#pragma unroll
    for (int i = 0; i < 32; ++i) emax = max(emax, (word(i) >> 7) & 0xffu);
#pragma unroll
    for (int o = 16; o; o >>= 1) emax = max(emax, __shfl_xor_sync(0xffffffffu, emax, o));
    const int base = (int)emax;
    uint32_t sm[8] = {}, codes[4] = {};
    int n_exc = 0;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        const uint32_t x = word(i);
        const int e = (int)((x >> 7) & 0xffu);
        sm[i >> 2] |= (((x >> 8) & 0x80u) | (x & 0x7fu)) << ((i & 3) * 8);
        const int c = e >= base - 14 ? e - base + 15 : 0;
        codes[i >> 3] |= (uint32_t)c << ((i & 7) * 4);
        n_exc += c == 0;
    }
    // exceptions: warp-wide prefix of the per-lane counts
    int pre = n_exc;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, pre, o);
        if (lane >= o) pre += t;
    }
    const int total = __shfl_sync(0xffffffffu, pre, 31);
    pre -= n_exc;  // exclusive
    uint8_t* dst = out + sb * kPackedSb;
    uint4* dsm = reinterpret_cast<uint4*>(dst + lane * 32);
    dsm[0] = make_uint4(sm[0], sm[1], sm[2], sm[3]);
    dsm[1] = make_uint4(sm[4], sm[5], sm[6], sm[7]);
    *reinterpret_cast<uint4*>(dst + 1024 + lane * 16) = make_uint4(codes[0], codes[1], codes[2], codes[3]);
    uint32_t* rec = reinterpret_cast<uint32_t*>(dst + 1536);
    if (lane >= 1 && lane < 8) rec[lane] = 0;  // unused entries: defined contents
    __syncwarp();
    if (total <= kPackMaxExc && n_exc) {
        int k = pre;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
            const uint32_t x = word(i);
            const int e = (int)((x >> 7) & 0xffu);
            if (e < base - 14) rec[1 + k++] = (uint32_t)(lane * 32 + i) | ((uint32_t)e << 16);
        }
    }
    if (lane == 0) {
        rec[0] = (uint32_t)base | ((uint32_t)(total <= kPackMaxExc ? total : 0xff) << 8);
        if (total > kPackMaxExc && raw_list) {  // carried raw: listed for the caller
            const uint32_t k = atomicAdd(raw_list, 1u);
            if (k < raw_cap) raw_list[1 + k] = first_sb + (uint32_t)sb;
        }
    }
}

__global__ void __launch_bounds__(256) unpack_kernel(const uint8_t* __restrict__ in, uint64_t n_sb,
                                                     uint16_t* __restrict__ out) {
    const uint64_t sb = (uint64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
    if (sb >= n_sb) return;
    const int lane = threadIdx.x & 31;
    const uint8_t* src = in + sb * kPackedSb;
    const uint32_t r = lane < 8 ? reinterpret_cast<const uint32_t*>(src + 1536)[lane] : 0u;
    const uint32_t head = __shfl_sync(0xffffffffu, r, 0);
    const int base = (int)(head & 0xffu), n_exc = (int)((head >> 8) & 0xffu);
    if (n_exc == 0xff) return;  // carried raw
    const uint4 s0 = reinterpret_cast<const uint4*>(src + lane * 32)[0];
    const uint4 s1 = reinterpret_cast<const uint4*>(src + lane * 32)[1];
    const uint4 cv = *reinterpret_cast<const uint4*>(src + 1024 + lane * 16);
    const uint32_t sm[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
    const uint32_t codes[4] = {cv.x, cv.y, cv.z, cv.w};
    uint32_t exc[kPackMaxExc];
#pragma unroll
    for (int k = 0; k < kPackMaxExc; ++k) exc[k] = __shfl_sync(0xffffffffu, r, 1 + k);
    uint32_t o[16];
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        const uint32_t b = (sm[i >> 2] >> ((i & 3) * 8)) & 0xffu;
        const int c = (int)((codes[i >> 3] >> ((i & 7) * 4)) & 0xfu);
        uint32_t e = (uint32_t)(base + c - 15);
        if (c == 0) {
            e = 0;
#pragma unroll
            for (int k = 0; k < kPackMaxExc; ++k)
                if (k < n_exc && (exc[k] & 0xffffu) == (uint32_t)(lane * 32 + i)) e = exc[k] >> 16;
        }
        const uint32_t x = ((b & 0x80u) << 8) | ((e & 0xffu) << 7) | (b & 0x7fu);
        if (i & 1)
            o[i >> 1] |= x << 16;
        else
            o[i >> 1] = x;
    }
    uint4* dst = reinterpret_cast<uint4*>(out + sb * kPackWords + lane * 32);
#pragma unroll
    for (int i = 0; i < 4; ++i) dst[i] = make_uint4(o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
}

}  // namespace

cudaError_t launch_pack(const uint16_t* in, uint64_t n_sb, uint8_t* out, uint32_t* raw_list, uint32_t first_sb,
                        uint32_t raw_cap, cudaStream_t st) {
    if (n_sb == 0) return cudaSuccess;
    if (((uintptr_t)in & 15) || ((uintptr_t)out & 15)) return cudaErrorInvalidValue;
    pack_kernel<<<(unsigned)((n_sb + kWarps - 1) / kWarps), 256, 0, st>>>(in, n_sb, out, raw_list, first_sb, raw_cap);
    return cudaGetLastError();
}

cudaError_t launch_unpack(const uint8_t* in, uint64_t n_sb, uint16_t* out, cudaStream_t st) {
    if (n_sb == 0) return cudaSuccess;
    if (((uintptr_t)in & 15) || ((uintptr_t)out & 15)) return cudaErrorInvalidValue;
    unpack_kernel<<<(unsigned)((n_sb + kWarps - 1) / kWarps), 256, 0, st>>>(in, n_sb, out);
    return cudaGetLastError();
}

}  // namespace loip
