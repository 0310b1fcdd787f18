// pack.cu -- lossless packing of bf16 weights for the host link.
//
// The streamed layers cross the host link every step, and the link is the
// step's bound, so the stream carries fewer bytes without changing a single
// weight: each bf16 word w = [sign | exponent (8) | mantissa (7)] is split into
// its sign-and-mantissa byte, stored as is, and its exponent, stored as a short
// code.  Within a superblock (1024 words) the exponents of model weights sit in
// a few binades below the largest one, a handful of them holding most words:
// with k = (largest exponent) - (exponent), the six most frequent k of the
// superblock get 2-bit codes in two levels, the other k up to 14 a 4-bit code,
// and anything else (zeros, values more than 14 binades down) is an exception
// listed in full.  For weights drawn like N(0, 0.02^2) that is ~2.7 bits per
// exponent where a plain code takes 4.  Decoding restores every word bit for bit.
//
// Packed superblock (kPackedSb = 1440 bytes for 1024 words = 2048 bytes):
//   bytes    0 .. 1023  sign-and-mantissa byte of word i: (w >> 8 & 0x80) | (w & 0x7f)
//   bytes 1024 .. 1279  level 1, 2 bits per word (word i: byte 1024 + i / 4, bits
//                       2 (i % 4)): c in 0..2: k = rank[c]; c = 3: go to level 2
//   bytes 1280 .. 1367  level 2, 2 bits per level-1 escape in word order (escape r:
//                       byte 1280 + r / 4, bits 2 (r % 4)): d in 0..2: k = rank[3 + d];
//                       d = 3: go to level 3 (at most kPackEsc1 level-1 escapes)
//   bytes 1368 .. 1407  level 3, 4 bits per level-2 escape in word order (escape s:
//                       byte 1368 + s / 2, low nibble for even s): v in 0..14: k = v;
//                       v = 15: an exception (at most kPackEsc2 level-2 escapes)
//   bytes 1408 .. 1439  record, 8 little-endian uint32: word 0 = emax | flag << 8 |
//                       rank[0] << 16 | rank[1] << 24 (flag 0: packed; 0xff: not
//                       packed -- over one of the limits -- every other byte of the
//                       superblock zero, and its 2048 raw bytes travel separately);
//                       word 1 = rank[2..5]; word 2 = n1 | n2 << 16 | n3 << 24 (the
//                       escape counts of levels 1 and 2 and the exception count, at
//                       most kPackMaxExc); words 3 + m: exception m = index | exponent << 16
// rank[0..5] are the six most frequent k in 0..14 of the superblock, most frequent
// first, ties to the smaller k.
//
// One warp per superblock in both directions; lane j handles words 8 j .. 8 j + 7
// of each quarter (256 words), so that every global load and store of a warp is
// one contiguous run.  A lane finds its first escape of each level with warp
// prefix sums over the word order (quarter, lane, word).
#include <cuda_runtime.h>
#include <stdint.h>

#include "internal.h"

namespace loip {
namespace {

constexpr int kWarps = 8;  // superblocks per 256-thread block
constexpr int kOffL1 = 1024, kOffL2 = 1280, kOffL3 = 1368, kOffRec = 1408;
static_assert(kOffRec + 32 == kPackedSb, "the record closes the superblock");
static_assert((kOffL3 - kOffL2) * 4 == kPackEsc1 && (kOffRec - kOffL3) * 2 == kPackEsc2, "stream areas");
static_assert(kOffRec - kOffL2 == 128, "levels 2 and 3 are one 32-word block");
static_assert(3 + kPackMaxExc <= 8, "exceptions fit the record");

__device__ __forceinline__ uint32_t word_of(const uint4& v, int e) {
    const uint32_t x = (e < 2) ? v.x : (e < 4) ? v.y : (e < 6) ? v.z : v.w;
    return (e & 1) ? x >> 16 : x & 0xffffu;
}

// exclusive warp prefix sum of n (lanes in order); *total gets the sum
__device__ __forceinline__ uint32_t warp_excl_scan(uint32_t n, int lane, uint32_t* total) {
    uint32_t s = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_up_sync(0xffffffffu, s, o);
        if (lane >= o) s += t;
    }
    *total = __shfl_sync(0xffffffffu, s, 31);
    return s - n;
}

__global__ void __launch_bounds__(256) pack_kernel(const uint16_t* __restrict__ in, uint64_t n_sb,
                                                   uint8_t* __restrict__ out, uint32_t* raw_list, uint32_t first_sb,
                                                   uint32_t raw_cap) {
    __shared__ uint32_t s_hist[kWarps][16];  // k histogram, then the exception entries
    __shared__ uint32_t s_bits[kWarps][32];  // levels 2 and 3 of the warp's superblock
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint64_t sb = (uint64_t)blockIdx.x * kWarps + warp;
    if (sb >= n_sb) return;  // warp-uniform; the kernel has no block-wide barrier
    uint4 w[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) w[q] = reinterpret_cast<const uint4*>(in + sb * kPackWords + 256 * q)[lane];
    uint32_t emax = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q)
#pragma unroll
        for (int e = 0; e < 8; ++e) emax = max(emax, (word_of(w[q], e) >> 7) & 0xffu);
#pragma unroll
    for (int o = 16; o; o >>= 1) emax = max(emax, __shfl_xor_sync(0xffffffffu, emax, o));
    // histogram of k (bin 15: k >= 15)
    if (lane < 16) s_hist[warp][lane] = 0;
    s_bits[warp][lane] = 0;
    __syncwarp();
#pragma unroll
    for (int q = 0; q < 4; ++q)
#pragma unroll
        for (int e = 0; e < 8; ++e) atomicAdd(&s_hist[warp][min(emax - ((word_of(w[q], e) >> 7) & 0xffu), 15u)], 1u);
    __syncwarp();
    const uint32_t cnt = lane < 15 ? s_hist[warp][lane] : 0u;
    __syncwarp();  // s_hist is reused for the exceptions below
    // the six most frequent k in 0..14, ties to the smaller k (lane b holds bin b)
    bool taken = lane >= 15;
    uint64_t ranks = 0;
#pragma unroll
    for (int i = 0; i < 6; ++i) {
        uint32_t key = taken ? 0u : ((cnt + 1u) << 8) | (255u - (uint32_t)lane);
#pragma unroll
        for (int o = 16; o; o >>= 1) key = max(key, __shfl_xor_sync(0xffffffffu, key, o));
        const uint32_t k = 255u - (key & 0xffu);
        ranks |= (uint64_t)k << (8 * i);
        if ((uint32_t)lane == k) taken = true;
    }
    auto rank_of = [&](uint32_t k) -> int {  // 6: not one of the six
        int r = 6;
#pragma unroll
        for (int i = 5; i >= 0; --i)
            if (((ranks >> (8 * i)) & 0xffu) == k) r = i;
        return r;
    };
    // level-1 codes and escape counts per quarter
    uint32_t c16[4], n1[4], n2[4], n3[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        c16[q] = 0;
        n1[q] = n2[q] = n3[q] = 0;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const uint32_t k = emax - ((word_of(w[q], e) >> 7) & 0xffu);
            const int r = rank_of(k);
            c16[q] |= (uint32_t)(r < 3 ? r : 3) << (2 * e);
            n1[q] += r >= 3;
            n2[q] += r >= 6;
            n3[q] += r >= 6 && k > 14;
        }
    }
    uint32_t off1[4], off2[4], off3[4], t1 = 0, t2 = 0, t3 = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint32_t a, b, c;
        off1[q] = t1 + warp_excl_scan(n1[q], lane, &a);
        off2[q] = t2 + warp_excl_scan(n2[q], lane, &b);
        off3[q] = t3 + warp_excl_scan(n3[q], lane, &c);
        t1 += a;
        t2 += b;
        t3 += c;
    }
    const bool packed = t1 <= (uint32_t)kPackEsc1 && t2 <= (uint32_t)kPackEsc2 && t3 <= (uint32_t)kPackMaxExc;
    if (packed) {
        // levels 2 and 3 into the warp's 32-word block (2-bit and 4-bit fields
        // never straddle a word), exceptions into s_hist
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint32_t i1 = off1[q], i2 = off2[q], i3 = off3[q];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const uint32_t ex = (word_of(w[q], e) >> 7) & 0xffu, k = emax - ex;
                const int r = rank_of(k);
                if (r < 3) continue;
                const uint32_t d = r < 6 ? (uint32_t)(r - 3) : 3u;
                atomicOr(&s_bits[warp][i1 >> 4], d << (2 * (i1 & 15)));
                ++i1;
                if (d < 3) continue;
                const uint32_t v = k <= 14 ? k : 15u;
                atomicOr(&s_bits[warp][22 + (i2 >> 3)], v << (4 * (i2 & 7)));
                ++i2;
                if (v < 15) continue;
                if (i3 < (uint32_t)kPackMaxExc) s_hist[warp][i3] = (256u * q + 8u * lane + e) | (ex << 16);
                ++i3;
            }
        }
    }
    __syncwarp();
    uint32_t rec = 0;  // lane j < 8: record word j
    if (packed) {
        if (lane == 0) rec = emax | ((uint32_t)(ranks & 0xffffu) << 16);
        if (lane == 1) rec = (uint32_t)(ranks >> 16);
        if (lane == 2) rec = t1 | (t2 << 16) | (t3 << 24);
        if (lane >= 3 && lane < 3 + kPackMaxExc && (uint32_t)(lane - 3) < t3) rec = s_hist[warp][lane - 3];
    } else if (lane == 0) {
        rec = emax | (0xffu << 8);
    }
    // stores: sign-and-mantissa bytes, level-1 codes, levels 2-3, record
    uint8_t* dst = out + sb * kPackedSb;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint32_t sm0 = 0, sm1 = 0;
        if (packed) {
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const uint32_t x = word_of(w[q], e), b = ((x >> 8) & 0x80u) | (x & 0x7fu);
                if (e < 4)
                    sm0 |= b << (8 * e);
                else
                    sm1 |= b << (8 * (e - 4));
            }
        }
        reinterpret_cast<uint2*>(dst + 256 * q)[lane] = make_uint2(sm0, sm1);
        reinterpret_cast<uint16_t*>(dst + kOffL1 + 64 * q)[lane] = (uint16_t)(packed ? c16[q] : 0u);
    }
    reinterpret_cast<uint32_t*>(dst + kOffL2)[lane] = packed ? s_bits[warp][lane] : 0u;
    if (lane < 8) reinterpret_cast<uint32_t*>(dst + kOffRec)[lane] = rec;
    if (!packed && lane == 0 && raw_list) {  // carried raw: listed for the caller
        const uint32_t k = atomicAdd(raw_list, 1u);
        if (k < raw_cap) raw_list[1 + k] = first_sb + (uint32_t)sb;
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
    uint32_t c16[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        sm[q] = __ldcs(reinterpret_cast<const uint2*>(src + 256 * q) + lane);
        c16[q] = __ldcs(reinterpret_cast<const unsigned short*>(src + kOffL1 + 64 * q) + lane);
    }
    const uint32_t lv = __ldcs(reinterpret_cast<const uint32_t*>(src + kOffL2) + lane);  // levels 2-3, word `lane`
    const uint32_t r = lane < 8 ? __ldcs(reinterpret_cast<const uint32_t*>(src + kOffRec) + lane) : 0u;
    const uint32_t r0 = __shfl_sync(0xffffffffu, r, 0);
    if (((r0 >> 8) & 0xffu) == 0xffu) return;  // carried raw
    const uint32_t emax = r0 & 0xffu;
    const uint64_t ranks = (uint64_t)(r0 >> 16) | ((uint64_t)__shfl_sync(0xffffffffu, r, 1) << 16);
    const uint32_t n_exc = __shfl_sync(0xffffffffu, r, 2) >> 24;
    // level-1 escapes per quarter (c = 3: both bits set), and each lane's first:
    // two quarters' counts per scan, in 16-bit halves (at most 256 per quarter)
    uint32_t n1[4], off1[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) n1[q] = __popc(c16[q] & (c16[q] >> 1) & 0x5555u);
    {
        uint32_t ta, tb;
        const uint32_t xa = warp_excl_scan(n1[0] | (n1[1] << 16), lane, &ta);
        const uint32_t xb = warp_excl_scan(n1[2] | (n1[3] << 16), lane, &tb);
        const uint32_t t0 = ta & 0xffffu, t1 = ta >> 16, t2 = tb & 0xffffu;
        off1[0] = xa & 0xffffu;
        off1[1] = t0 + (xa >> 16);
        off1[2] = t0 + t1 + (xb & 0xffffu);
        off1[3] = t0 + t1 + t2 + (xb >> 16);
    }
    // this lane's level-2 codes (at most 8 per quarter: 16 bits of a 2-word window)
    uint32_t l2[4], n2[4], off2[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint32_t wi = off1[q] >> 4, sh = 2 * (off1[q] & 15);
        const uint32_t lo = __shfl_sync(0xffffffffu, lv, (int)wi & 31);
        const uint32_t hi = __shfl_sync(0xffffffffu, lv, (int)(wi + 1) & 31);
        l2[q] = __funnelshift_r(lo, hi, sh) & (n1[q] ? 0xffffu >> (16 - 2 * n1[q]) : 0u);
        n2[q] = __popc(l2[q] & (l2[q] >> 1) & 0x5555u);
    }
    {
        uint32_t ta, tb;
        const uint32_t xa = warp_excl_scan(n2[0] | (n2[1] << 16), lane, &ta);
        const uint32_t xb = warp_excl_scan(n2[2] | (n2[3] << 16), lane, &tb);
        const uint32_t t0 = ta & 0xffffu, t1 = ta >> 16, t2 = tb & 0xffffu;
        off2[0] = xa & 0xffffu;
        off2[1] = t0 + (xa >> 16);
        off2[2] = t0 + t1 + (xb & 0xffffu);
        off2[3] = t0 + t1 + t2 + (xb >> 16);
    }
    // k of four words at once: the level-1 codes select bytes of the first three
    // ranks; code 3 selects 0xff, which marks the escapes (no k is above 14)
    const uint32_t R1 = (uint32_t)(ranks & 0xffffffu) | 0xff000000u;
    const uint32_t R2 = (uint32_t)((ranks >> 24) & 0xffffffu) | 0xff000000u;  // ranks 3..5, 0xff: level 3
    const uint32_t E4 = emax * 0x01010101u;
    // 2-bit fields at bits 2j -> 4-bit fields at bits 4j (j < 8)
    auto spread2 = [](uint32_t v) -> uint32_t {
        v = (v | (v << 8)) & 0x00ff00ffu;
        v = (v | (v << 4)) & 0x0f0f0f0fu;
        return (v | (v << 2)) & 0x33333333u;
    };
    uint4 o[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint32_t sel = spread2(c16[q]);  // nibble e = level-1 code of word e
        uint32_t k03 = __byte_perm(R1, 0u, sel), k47 = __byte_perm(R1, 0u, sel >> 16);
        // level 2 without a loop: T holds, for the lane's j-th escape of the
        // quarter, the k its level-2 code names (0xff: level 3); escape word e
        // takes entry rank(e), the number of escapes before it (a nibble-wise
        // prefix product)
        const uint32_t escN = sel & (sel >> 1) & 0x11111111u;  // nibble e = 1: word e escapes
        const uint32_t rk = escN * 0x11111111u - escN;
        const uint32_t t4 = spread2(l2[q]);  // nibble j = the j-th level-2 code
        const uint32_t T0 = __byte_perm(R2, 0u, t4), T1 = __byte_perm(R2, 0u, t4 >> 16);
        const uint32_t M03 = ((k03 & 0x80808080u) >> 7) * 0xffu, M47 = ((k47 & 0x80808080u) >> 7) * 0xffu;
        k03 = (k03 & ~M03) | (__byte_perm(T0, T1, rk & 0x7777u) & M03);
        k47 = (k47 & ~M47) | (__byte_perm(T0, T1, (rk >> 16) & 0x7777u) & M47);
        // level 3 (rare): the words still marked 0xff, in word order; this lane's
        // nibbles of the quarter (at most 8: a 2-word window of words 22..31,
        // shuffled by the whole warp)
        const uint32_t wi = 22 + (off2[q] >> 3), sh = 4 * (off2[q] & 7);
        const uint32_t lo = __shfl_sync(0xffffffffu, lv, (int)wi & 31);
        const uint32_t hi = __shfl_sync(0xffffffffu, lv, (int)(wi + 1) & 31);
        uint32_t m03 = k03 & 0x80808080u, m47 = k47 & 0x80808080u;
        if (m03 | m47) {
            uint32_t l3 = wi < 32 ? __funnelshift_r(lo, wi + 1 < 32 ? hi : 0u, sh) : 0u;
            while (m03) {
                const uint32_t shb = (uint32_t)(__ffs(m03) - 8);  // 8 * byte
                m03 &= m03 - 1;
                k03 = (k03 & ~(0xffu << shb)) | ((l3 & 15u) << shb);  // 15: an exception, patched below
                l3 >>= 4;
            }
            while (m47) {
                const uint32_t shb = (uint32_t)(__ffs(m47) - 8);
                m47 &= m47 - 1;
                k47 = (k47 & ~(0xffu << shb)) | ((l3 & 15u) << shb);
                l3 >>= 4;
            }
        }
        // exponent bytes: emax - k never borrows (k <= emax; the exception
        // placeholder 15 only where emax >= 15)
        const uint32_t x03 = E4 - k03, x47 = E4 - k47;
        // two words per register: sign | exponent << 7 | mantissa
        auto pair = [](uint32_t smb, uint32_t xb, uint32_t sel2) -> uint32_t {
            const uint32_t t = __byte_perm(smb, 0u, sel2), ee = __byte_perm(xb, 0u, sel2);
            return ((t & 0x00800080u) << 8) | (ee << 7) | (t & 0x007f007fu);
        };
        o[q] = make_uint4(pair(sm[q].x, x03, 0x4140u), pair(sm[q].x, x03, 0x4342u), pair(sm[q].y, x47, 0x4140u),
                          pair(sm[q].y, x47, 0x4342u));
    }
    // exceptions, into the register of the lane that holds the word
    for (uint32_t m = 0; m < n_exc; ++m) {
        const uint32_t x = __shfl_sync(0xffffffffu, r, 3 + (int)m);
        const uint32_t idx = x & 0xffffu;
        if (((idx >> 3) & 31u) != (uint32_t)lane) continue;
        const uint32_t quarter = idx >> 8, e = idx & 7u, sh = 7 + 16 * (e & 1u);
        const uint32_t keep = ~(0xffu << sh), v = ((x >> 16) & 0xffu) << sh;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            if ((uint32_t)q != quarter) continue;
            if ((e >> 1) == 0) o[q].x = (o[q].x & keep) | v;
            if ((e >> 1) == 1) o[q].y = (o[q].y & keep) | v;
            if ((e >> 1) == 2) o[q].z = (o[q].z & keep) | v;
            if ((e >> 1) == 3) o[q].w = (o[q].w & keep) | v;
        }
    }
    uint4* dst = reinterpret_cast<uint4*>(out + sb * kPackWords) + lane;
#pragma unroll
    for (int q = 0; q < 4; ++q) __stcs(dst + 32 * q, o[q]);  // streamed out: not read again soon
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
