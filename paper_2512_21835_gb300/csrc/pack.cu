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
// One warp per superblock in both directions; in the pack kernel lane j handles
// words 32 j .. 32 j + 31.
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

// Unpack: lane j of the warp takes words 8j .. 8j + 7 of each quarter (256
// words) of the superblock, so every load and store of the warp is one
// contiguous run (256 sign-and-mantissa bytes, 128 code bytes, 512 output
// bytes); the words are rebuilt two at a time in 32-bit registers.
__device__ __forceinline__ uint32_t unpack_pair(uint32_t sm4, uint32_t sel, uint32_t code_byte, uint32_t add) {
    const uint32_t t = __byte_perm(sm4, 0u, sel);                // byte b0 | byte b1 << 16
    const uint32_t n = __byte_perm(code_byte, 0u, 0x4040u);      // the two codes, in both halves
    uint32_t e = (n & 0x0000000fu) | ((n >> 4) & 0x000f0000u);   // code of word 0 | code of word 1 << 16
    e = (e + add) & 0x00ff00ffu;                                 // base + code - 15, modulo 256, per half
    return ((t & 0x00800080u) << 8) | (e << 7) | (t & 0x007f007fu);
}

// Exception k of the superblock (word index | exponent << 16) into the register
// of the lane that holds the word.
__device__ __forceinline__ void unpack_patch(uint4 (&o)[4], int lane, uint32_t x) {
    const int idx = (int)(x & 0xffffu);
    if (((idx >> 3) & 31) != lane) return;
    const int quarter = idx >> 8, q = idx & 7;
    const int sh = 7 + 16 * (q & 1);
    const uint32_t keep = ~(0xffu << sh), v = ((x >> 16) & 0xffu) << sh;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        if (k != quarter) continue;
        if ((q >> 1) == 0) o[k].x = (o[k].x & keep) | v;
        if ((q >> 1) == 1) o[k].y = (o[k].y & keep) | v;
        if ((q >> 1) == 2) o[k].z = (o[k].z & keep) | v;
        if ((q >> 1) == 3) o[k].w = (o[k].w & keep) | v;
    }
}

// One launch unpacks one or two segments (runs of superblocks, each with its
// own input and output): blocks [0, s0.blocks) take the first, the rest the
// second.  Two chunks per launch halve the launches, whose start-up after an
// idle wait for the host link costs about as much as the unpack itself.
struct UnpackSeg {
    const uint8_t* in;
    uint16_t* out;
    uint64_t n_sb;
    uint32_t blocks;
};

__global__ void __launch_bounds__(256) unpack_kernel(UnpackSeg s0, UnpackSeg s1) {
    const bool second = blockIdx.x >= s0.blocks;
    const uint8_t* __restrict__ in = second ? s1.in : s0.in;
    uint16_t* __restrict__ out = second ? s1.out : s0.out;
    const uint64_t sb = (uint64_t)(blockIdx.x - (second ? s0.blocks : 0u)) * kWarps + (threadIdx.x >> 5);
    if (sb >= (second ? s1.n_sb : s0.n_sb)) return;
    const int lane = threadIdx.x & 31;
    const uint8_t* src = in + sb * kPackedSb;
    // every load first: read once, evict first
    uint2 sm[4];
    uint32_t codes[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        sm[k] = __ldcs(reinterpret_cast<const uint2*>(src + 256 * k) + lane);
        codes[k] = __ldcs(reinterpret_cast<const uint32_t*>(src + 1024 + 128 * k) + lane);
    }
    const uint32_t r = lane < 8 ? __ldcs(reinterpret_cast<const uint32_t*>(src + 1536) + lane) : 0u;
    const uint32_t head = __shfl_sync(0xffffffffu, r, 0);
    const uint32_t base = head & 0xffu, n_exc = (head >> 8) & 0xffu;
    if (n_exc == 0xffu) return;  // carried raw
    const uint32_t add = ((base + 241u) & 0xffu) * 0x10001u;  // 241 = -15 modulo 256
    uint4 o[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        o[k].x = unpack_pair(sm[k].x, 0x4140u, codes[k], add);
        o[k].y = unpack_pair(sm[k].x, 0x4342u, codes[k] >> 8, add);
        o[k].z = unpack_pair(sm[k].y, 0x4140u, codes[k] >> 16, add);
        o[k].w = unpack_pair(sm[k].y, 0x4342u, codes[k] >> 24, add);
    }
    for (uint32_t k = 0; k < n_exc; ++k) unpack_patch(o, lane, __shfl_sync(0xffffffffu, r, 1 + k));
    uint4* dst = reinterpret_cast<uint4*>(out + sb * kPackWords) + lane;
#pragma unroll
    for (int k = 0; k < 4; ++k) __stcs(dst + 32 * k, o[k]);  // streamed out: not read again soon
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
    return launch_unpack2(in, n_sb, out, nullptr, 0, nullptr, st);
}

cudaError_t launch_unpack2(const uint8_t* in0, uint64_t n0, uint16_t* out0, const uint8_t* in1, uint64_t n1,
                           uint16_t* out1, cudaStream_t st) {
    if (n0 + n1 == 0) return cudaSuccess;
    if (((uintptr_t)in0 & 15) || ((uintptr_t)out0 & 15) || ((uintptr_t)in1 & 15) || ((uintptr_t)out1 & 15))
        return cudaErrorInvalidValue;
    const UnpackSeg s0{in0, out0, n0, (uint32_t)((n0 + kWarps - 1) / kWarps)};
    const UnpackSeg s1{in1, out1, n1, (uint32_t)((n1 + kWarps - 1) / kWarps)};
    unpack_kernel<<<s0.blocks + s1.blocks, 256, 0, st>>>(s0, s1);
    return cudaGetLastError();
}

}  // namespace loip
