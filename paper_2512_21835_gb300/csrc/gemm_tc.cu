// gemm_tc.cu -- prefill projections on the 5th-generation tensor cores.
//
// C[M, N] = A[M, K] * W[N, K]^T with A the activations of M prompt tokens and
// W a bf16 weight matrix (both K-contiguous), fp32 accumulation in tensor
// memory, fused epilogues (query/key rotation + KV-cache write, residual add,
// SwiGLU).
//
// Activations are fp32 on this path; the tensor cores take bf16 operands of
// one type (kind::f16).  So an activation matrix is given as a pair of bf16
// planes, A = A_hi + A_lo with A_hi = bf16(A) and A_lo = bf16(A - A_hi) (a
// "split" operand, ~16 significant bits), and every K step issues two MMAs
// into the same accumulator: A_hi W^T and A_lo W^T.  The weights are the
// model's unmodified bf16 values, so the product equals the fp32-activation
// product up to fp32 accumulation and the 2^-17 relative residue of the pair.
// A single bf16 plane (no split) is also supported.
//
// Output tiles are 128 x 256, computed by a persistent grid (one CTA per SM,
// tiles rasterised M-fastest):
//   warp 0     TMA producer: a ring of stages (A_hi [, A_lo] 128x64 and W
//              256x64, bf16, 128-byte swizzle; 4 stages of 48 KB, or 3 of
//              64 KB when split), one mbarrier per stage with transaction bytes;
//   warp 1     allocates 512 TMEM columns (two accumulators), one lane issues
//              tcgen05.mma (M 128, N 256, K 16) and frees a stage with
//              tcgen05.commit;
//   warps 2-9  drain the accumulators chunk by chunk into fp32 registers and
//              run the fused epilogue (two warps per 32-lane TMEM quadrant, one
//              output row per thread, half of the tile's columns each).
// Every mbarrier wait is bounded; on timeout the kernel records an error code,
// every role of the CTA stops, copies and MMAs in flight finish, TMEM is freed
// and the kernel returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "internal.h"

namespace loip {

__device__ int g_tc_error;  // first failure code of any tensor-core GEMM launch (0 = none)

namespace {

constexpr int TBM = 128, TBN = 256, TBK = 64;
constexpr int A_BYTES = TBM * TBK * 2;          // 16 KB: one plane of the A tile
constexpr int B_HALF = 128 * TBK * 2;           // 16 KB: one 128-row TMA box of W
template <int SPLIT>
struct Ring {
    static constexpr int STAGES = SPLIT ? 3 : 4;
    static constexpr int B_OFF = (SPLIT ? 2 : 1) * A_BYTES;  // W tile after the A plane(s)
    static constexpr int STAGE_BYTES = B_OFF + 2 * B_HALF;
    static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + 256;
};
// instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, N = 256, M = 128
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(TBN >> 3) << 17) |
                            ((uint32_t)(TBM >> 4) << 24);

enum { T_QKV = 0, T_RESID = 1, T_SWIGLU = 2 };

struct TcParams {
    int M, N, K;  // N: output columns (QKV, RESID) or F (SWIGLU)
    int n_tiles;  // output tiles along N
    float* x;
    uint16_t* a;  // SWIGLU output: split pair [2][M][N] (hi plane, then lo plane)
    float* q;
    int Hq, Hkv, d;
    const int32_t* positions;
    const int32_t* row_req;
    KvView kv;
    RopeFreqs rope;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
// Wait for the phase with the given parity.  try_wait suspends the thread in
// hardware for a bounded, system-defined time per call, so waiting warps do not
// take issue slots from the producer and MMA warps; the loop gives up after 2 s
// of wall time.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (global_ns() - t0 > 2000000000ull) return false;
    }
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            dst),
        "l"((uint64_t)map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
            tmem_d),
        "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
// Shared-memory matrix descriptor: K-major operand, rows of 128 bytes with the
// 128-byte swizzle, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)1 << 16;              // leading byte offset (unused for this layout)
    d |= (uint64_t)(1024 >> 4) << 32;    // stride byte offset
    d |= (uint64_t)1 << 46;              // descriptor version
    d |= (uint64_t)2 << 61;              // 128-byte swizzle
    return d;
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%"
        "19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
          "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ uint16_t f2bf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }
__device__ __forceinline__ float bf2f(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }

__device__ __forceinline__ void record_error(int code) { atomicCAS(&g_tc_error, 0, code); }

// ----------------------------------------------------------------------------
// Epilogues from registers.  Epilogue warp w (2..9) owns TMEM lane quadrant
// q = w % 4 (its rows 32 q .. 32 q + 31 of the tile, one row per lane) and
// half h = (w - 2) / 4 of the tile's columns; acc[] holds that thread's 128
// fp32 sums.  Column sets (so that each thread holds what its epilogue pairs):
//   RESID, QKV: columns [128 h, 128 h + 128) (whole heads: RoPE pairs i, i + d/2
//               sit inside a head, and d divides 128);
//   SWIGLU:     gate columns [64 h, 64 h + 64) and the matching up columns
//               [128 + 64 h, 128 + 64 h + 64) (the tile's gate rows 0..127 of
//               W_g, up rows 128..255 of W_u).
// ----------------------------------------------------------------------------
template <int EPI>
__device__ __forceinline__ int col_of(int h, int j) {  // tile column of acc[j]
    if (EPI == T_SWIGLU) return j < 64 ? 64 * h + j : 128 + 64 * h + (j - 64);
    return 128 * h + j;
}

__device__ __forceinline__ void epi_resid(const TcParams& p, const float (&acc)[128], int row, int c0) {
    float* xr = p.x + (size_t)row * p.N + c0;
    if (c0 + 128 <= p.N) {
#pragma unroll
        for (int j = 0; j < 128; j += 4) {
            float4 t = *reinterpret_cast<float4*>(xr + j);
            t.x += acc[j];
            t.y += acc[j + 1];
            t.z += acc[j + 2];
            t.w += acc[j + 3];
            *reinterpret_cast<float4*>(xr + j) = t;
        }
    } else {
#pragma unroll
        for (int j = 0; j < 128; ++j)
            if (c0 + j < p.N) xr[j] += acc[j];
    }
}

// silu(g) * u, written as the split pair (hi plane, lo plane M * F further on)
__device__ __forceinline__ void epi_swiglu(const TcParams& p, const float (&acc)[128], int row, int f0) {
    uint16_t* ar = p.a + (size_t)row * p.N + f0;
    const size_t plane = (size_t)p.M * p.N;
    if (f0 + 64 <= p.N) {
#pragma unroll
        for (int j = 0; j < 64; j += 8) {
            uint32_t w[4], wl[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float g0 = acc[j + 2 * e], g1 = acc[j + 2 * e + 1];
                const float s0 = g0 / (1.0f + expf(-g0)) * acc[64 + j + 2 * e];
                const float s1 = g1 / (1.0f + expf(-g1)) * acc[64 + j + 2 * e + 1];
                const uint16_t h0 = f2bf(s0), h1 = f2bf(s1);
                w[e] = (uint32_t)h0 | ((uint32_t)h1 << 16);
                wl[e] = (uint32_t)f2bf(s0 - bf2f(h0)) | ((uint32_t)f2bf(s1 - bf2f(h1)) << 16);
            }
            *reinterpret_cast<uint4*>(ar + j) = make_uint4(w[0], w[1], w[2], w[3]);
            *reinterpret_cast<uint4*>(ar + plane + j) = make_uint4(wl[0], wl[1], wl[2], wl[3]);
        }
    } else {
#pragma unroll
        for (int j = 0; j < 64; ++j)
            if (f0 + j < p.N) {
                const float g = acc[j];
                const float sv = g / (1.0f + expf(-g)) * acc[64 + j];
                const uint16_t h = f2bf(sv);
                ar[j] = h;
                ar[plane + j] = f2bf(sv - bf2f(h));
            }
    }
}

// QKV columns c0 .. c0 + 127 (128 / D whole heads): rotate query and key heads
// at the row's position, store queries fp32 and keys / values bf16 in the page.
template <int D>
__device__ __forceinline__ void epi_qkv(const TcParams& p, float (&acc)[128], int row, int c0) {
    constexpr int HALF = D / 2;
    const int pos = p.positions[row];
#pragma unroll
    for (int hc = 0; hc < 128; hc += D) {
        if (c0 + hc >= p.N) break;  // uniform across the warp
        const int h = (c0 + hc) / D;
        if (h < p.Hq + p.Hkv) {
#pragma unroll
            for (int i = 0; i < HALF; ++i) {
                float c, s;
                rope_cos_sin(pos, p.rope.inv_freq[i], &c, &s);
                const float v0 = acc[hc + i], v1 = acc[hc + HALF + i];
                acc[hc + i] = v0 * c - v1 * s;
                acc[hc + HALF + i] = v1 * c + v0 * s;
            }
        }
        if (h < p.Hq) {
            float* qr = p.q + (size_t)row * p.Hq * D + (size_t)h * D;
#pragma unroll
            for (int j = 0; j < D; j += 4)
                *reinterpret_cast<float4*>(qr + j) = make_float4(acc[hc + j], acc[hc + j + 1], acc[hc + j + 2],
                                                                 acc[hc + j + 3]);
        } else {
            const bool is_v = h >= p.Hq + p.Hkv;
            const int kh = h - p.Hq - (is_v ? p.Hkv : 0);
            const int req = p.row_req[row];
            const int page = pos / p.kv.page_tokens, t = pos - page * p.kv.page_tokens;
            char* base = p.kv.base + p.kv.page_offsets[(int64_t)req * p.kv.max_pages + page] +
                         (uint64_t)p.kv.layer * p.kv.layer_page_bytes;
            uint16_t* kr = reinterpret_cast<uint16_t*>(
                base + ((uint64_t)((is_v ? p.Hkv : 0) + kh) * p.kv.page_tokens + t) * (uint64_t)D * 2u);
#pragma unroll
            for (int j = 0; j < D; j += 8) {
                uint32_t w[4];
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    w[e] = (uint32_t)f2bf(acc[hc + j + 2 * e]) | ((uint32_t)f2bf(acc[hc + j + 2 * e + 1]) << 16);
                *reinterpret_cast<uint4*>(kr + j) = make_uint4(w[0], w[1], w[2], w[3]);
            }
        }
    }
}

// Bounded wait that also leaves once another role of the CTA has aborted.
__device__ __forceinline__ bool mbar_wait_ab(uint32_t bar, uint32_t parity, volatile int* abort) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort) return false;
        if (global_ns() - t0 > 2000000000ull) {
            *abort = 1;
            return false;
        }
    }
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// Persistent tensor-core GEMM.  CTA b takes output tiles b, b + grid, ... in
// M-fastest order (the CTAs sharing a weight tile run together, so it is read
// from HBM about once).  Roles:
//   warp 0      TMA producer over every k-block of every tile (one smem ring);
//   warp 1      allocates the 512 TMEM columns (two 128 x 256 fp32
//               accumulators) and issues the MMAs.  The K range of a tile is cut
//               into chunks of KC k-blocks; chunk g of the CTA accumulates into
//               buffer g % 2 from zero;
//   warps 2-9   drain each finished chunk from TMEM into fp32 registers
//               (round-to-nearest adds), release the buffer, and after a tile's
//               last chunk run its epilogue from the registers -- while the MMAs
//               of the next chunk or tile already run on the other buffer.
// The tensor core's own accumulation truncates (its error grows with the
// number of MMAs summed into one accumulator, biased toward zero); summing at
// most KC k-blocks there and the chunks in fp32 keeps the product at fp32-GEMV
// accuracy.
constexpr int kEpiWarps = 8;
constexpr int kThreadsTC = 64 + 32 * kEpiWarps;
constexpr uint32_t kTmemCols = 512;
constexpr int KC = 16;  // k-blocks per accumulation chunk (K = 1024)

// 10 warps: the SM's four register partitions (16K each) hold three warps in
// two of them, so at most 168 registers per thread -- enough for an epilogue
// thread's 128 fp32 running sums (a few words spill around the epilogue)
template <int EPI, int SPLIT>
__global__ void __launch_bounds__(kThreadsTC, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmAlo,
                   const __grid_constant__ CUtensorMap tmB0, const __grid_constant__ CUtensorMap tmB1, TcParams p) {
    constexpr int STAGES = Ring<SPLIT>::STAGES, STAGE_BYTES = Ring<SPLIT>::STAGE_BYTES, B_OFF = Ring<SPLIT>::B_OFF;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
    // bars: full[STAGES], empty[STAGES], cfull[2], cempty[2], mma_done
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 5);
    volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m_tiles = (p.M + TBM - 1) / TBM;
    const int n_total = m_tiles * p.n_tiles;
    const int nk = (p.K + TBK - 1) / TBK;
    const int nchunks = (nk + KC - 1) / KC;
    const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + STAGES);
    const uint32_t cfull0 = smem_u32(bars + 2 * STAGES), cempty0 = smem_u32(bars + 2 * STAGES + 2);
    const uint32_t done_bar = smem_u32(bars + 2 * STAGES + 4);

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(cfull0 + 8 * b, 1);
            mbar_init(cempty0 + 8 * b, kEpiWarps);
        }
        mbar_init(done_bar, 1);
        *abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            const CUtensorMap* mb1 = (EPI == T_SWIGLU) ? &tmB1 : &tmB0;
            int kbg = 0;  // k-blocks issued by this CTA, over all its tiles
            for (int t = blockIdx.x; t < n_total && !*abort; t += gridDim.x) {
                const int m0 = (t % m_tiles) * TBM, ntile = t / m_tiles;
                const int y0 = (EPI == T_SWIGLU) ? ntile * 128 : ntile * TBN;
                const int y1 = (EPI == T_SWIGLU) ? ntile * 128 : ntile * TBN + 128;
                for (int kb = 0; kb < nk; ++kb, ++kbg) {
                    const int s = kbg % STAGES;
                    if (!mbar_wait_ab(empty0 + 8 * s, ((kbg / STAGES) & 1) ^ 1, abort)) {
                        record_error(1);
                        break;
                    }
                    const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
                    mbar_expect_tx(full0 + 8 * s, STAGE_BYTES);
                    tma_load_2d(sa, &tmA, kb * TBK, m0, full0 + 8 * s);
                    if (SPLIT) tma_load_2d(sa + A_BYTES, &tmAlo, kb * TBK, m0, full0 + 8 * s);
                    tma_load_2d(sa + B_OFF, &tmB0, kb * TBK, y0, full0 + 8 * s);
                    tma_load_2d(sa + B_OFF + B_HALF, mb1, kb * TBK, y1, full0 + 8 * s);
                }
            }
            // the copies of the last stages must land before this CTA's shared
            // memory can be released (bounded, and regardless of an abort)
            for (int k = kbg - STAGES < 0 ? 0 : kbg - STAGES; k < kbg; ++k)
                if (!mbar_wait(full0 + 8 * (k % STAGES), (k / STAGES) & 1)) record_error(4);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            int kbg = 0, cg = 0;  // k-blocks and chunks consumed by this CTA
            bool ok = true;
            for (int t = blockIdx.x; t < n_total && ok; t += gridDim.x) {
                for (int c = 0; c < nchunks && ok; ++c, ++cg) {
                    const int b = cg & 1;
                    if (!mbar_wait_ab(cempty0 + 8 * b, ((cg >> 1) & 1) ^ 1, abort)) {  // drained by the epilogue
                        record_error(5);
                        ok = false;
                        break;
                    }
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const uint32_t acc = tmem + (uint32_t)(b * TBN);
                    const int kb1 = (c + 1) * KC < nk ? (c + 1) * KC : nk;
                    for (int kb = c * KC; kb < kb1; ++kb, ++kbg) {
                        const int s = kbg % STAGES;
                        if (!mbar_wait_ab(full0 + 8 * s, (kbg / STAGES) & 1, abort)) {
                            record_error(2);
                            ok = false;
                            break;
                        }
                        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                        const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
                        const uint64_t da = smem_desc(sa), db = smem_desc(sa + B_OFF);
#pragma unroll
                        for (int k = 0; k < TBK / 16; ++k) {  // 32 bytes along K per instruction
                            umma_bf16(acc, da + 2 * k, db + 2 * k, (kb != c * KC || k != 0) ? 1u : 0u);
                            if (SPLIT) umma_bf16(acc, smem_desc(sa + A_BYTES) + 2 * k, db + 2 * k, 1u);  // + A_lo W^T
                        }
                        umma_commit(empty0 + 8 * s);
                    }
                    if (ok) umma_commit(cfull0 + 8 * b);  // the chunk is complete in buffer b
                }
            }
            // every MMA issued above completes before TMEM can be released
            umma_commit(done_bar);
            if (!mbar_wait(done_bar, 0)) record_error(6);
        }
        __syncwarp();
    } else {
        const int q = warp & 3, h = (warp - 2) >> 2;  // TMEM lane quadrant, column half
        int cg = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < n_total && ok; t += gridDim.x) {
            const int m0 = (t % m_tiles) * TBM, ntile = t / m_tiles;
            const int row = m0 + q * 32 + lane;
            float acc[128];
#pragma unroll
            for (int j = 0; j < 128; ++j) acc[j] = 0.f;
            for (int c = 0; c < nchunks; ++c, ++cg) {
                const int b = cg & 1;
                if (!mbar_wait_ab(cfull0 + 8 * b, (cg >> 1) & 1, abort)) {
                    record_error(3);
                    ok = false;
                    break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t tb = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * TBN);
#pragma unroll
                for (int j0 = 0; j0 < 128; j0 += 16) {
                    float v[16];
                    tmem_ld16(tb + (uint32_t)col_of<EPI>(h, j0), v);
#pragma unroll
                    for (int j = 0; j < 16; ++j) acc[j0 + j] += v[j];
                }
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(cempty0 + 8 * b);
            }
            if (!ok || row >= p.M) continue;
            if (EPI == T_RESID) {
                epi_resid(p, acc, row, ntile * TBN + 128 * h);
            } else if (EPI == T_SWIGLU) {
                epi_swiglu(p, acc, row, ntile * 128 + 64 * h);
            } else {
                if (p.d == 128)
                    epi_qkv<128>(p, acc, row, ntile * TBN + 128 * h);
                else
                    epi_qkv<64>(p, acc, row, ntile * TBN + 128 * h);
            }
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

cudaError_t encoder() {
    if (g_encode) return cudaSuccess;
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return cudaSuccess;
}

// 2-D map of a row-major [rows, K] bf16 matrix, box 64 (K) x 128 rows.
cudaError_t make_map(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t K) {
    if (((uintptr_t)ptr & 15) || (K * 2) % 16) return cudaErrorInvalidValue;
    cuuint64_t dims[2] = {K, rows};
    cuuint64_t strides[1] = {K * 2};
    cuuint32_t box[2] = {(cuuint32_t)TBK, 128};
    cuuint32_t es[2] = {1, 1};
    CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <int EPI, int SPLIT>
cudaError_t launch_tc_t(const void* A, const void* W0, const void* W1, uint64_t w_rows, TcParams& p, int n_tiles,
                        cudaStream_t st) {
    cudaError_t e = encoder();
    if (e != cudaSuccess) return e;
    if (p.M <= 0 || n_tiles <= 0) return cudaSuccess;
    CUtensorMap ma, malo, mb0, mb1;
    const uint16_t* A16 = static_cast<const uint16_t*>(A);
    if ((e = make_map(&ma, A16, (uint64_t)p.M, (uint64_t)p.K)) != cudaSuccess) return e;
    // the lo plane follows the hi plane (M * K elements on)
    if ((e = make_map(&malo, SPLIT ? A16 + (size_t)p.M * p.K : A16, (uint64_t)p.M, (uint64_t)p.K)) != cudaSuccess)
        return e;
    if ((e = make_map(&mb0, W0, w_rows, (uint64_t)p.K)) != cudaSuccess) return e;
    if ((e = make_map(&mb1, W1 ? W1 : W0, w_rows, (uint64_t)p.K)) != cudaSuccess) return e;
    constexpr int SMEM = Ring<SPLIT>::SMEM_BYTES;
    static bool attr = false;
    if (!attr) {
        e = cudaFuncSetAttribute(tc_gemm_kernel<EPI, SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    // persistent: one CTA per SM (the ring takes most of the shared memory), at
    // most one per tile
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
        if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    }
    p.n_tiles = n_tiles;
    const int tiles = ((p.M + TBM - 1) / TBM) * n_tiles;
    tc_gemm_kernel<EPI, SPLIT><<<tiles < sms ? tiles : sms, kThreadsTC, SMEM, st>>>(ma, malo, mb0, mb1, p);
    return cudaGetLastError();
}

template <int EPI>
cudaError_t launch_tc(const void* A, bool split, const void* W0, const void* W1, uint64_t w_rows, TcParams& p,
                      int n_tiles, cudaStream_t st) {
    return split ? launch_tc_t<EPI, 1>(A, W0, W1, w_rows, p, n_tiles, st)
                 : launch_tc_t<EPI, 0>(A, W0, W1, w_rows, p, n_tiles, st);
}

}  // namespace

cudaError_t launch_tc_gemm_qkv_rope(const uint16_t* y, bool split, const uint16_t* wqkv, int M, int H, int Hq,
                                    int Hkv, int d, float theta, const int32_t* positions, const int32_t* row_req,
                                    float* q, KvView kv, cudaStream_t st) {
    if (TBN % d != 0) return cudaErrorInvalidValue;
    TcParams p{};
    p.M = M;
    p.N = (Hq + 2 * Hkv) * d;
    p.K = H;
    p.q = q;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.d = d;
    p.positions = positions;
    p.row_req = row_req;
    p.kv = kv;
    p.rope = rope_freqs(theta, d);
    return launch_tc<T_QKV>(y, split, wqkv, nullptr, (uint64_t)p.N, p, (p.N + TBN - 1) / TBN, st);
}

cudaError_t launch_tc_gemm_resid(const uint16_t* a, bool split, const uint16_t* w, int M, int N, int K, float* x,
                                 cudaStream_t st) {
    TcParams p{};
    p.M = M;
    p.N = N;
    p.K = K;
    p.x = x;
    return launch_tc<T_RESID>(a, split, w, nullptr, (uint64_t)N, p, (N + TBN - 1) / TBN, st);
}

cudaError_t launch_tc_gemm_swiglu(const uint16_t* y, bool split, const uint16_t* wg, const uint16_t* wu, int M, int H,
                                  int F, uint16_t* a, cudaStream_t st) {
    TcParams p{};
    p.M = M;
    p.N = F;
    p.K = H;
    p.a = a;
    return launch_tc<T_SWIGLU>(y, split, wg, wu, (uint64_t)F, p, (F + 127) / 128, st);
}

cudaError_t tc_error(int* code) {
    return cudaMemcpyFromSymbol(code, g_tc_error, sizeof(int));
}

}  // namespace loip
