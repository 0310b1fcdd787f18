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
// One CTA computes a 128 x 256 output tile:
//   warp 0     TMA producer: a ring of stages (A_hi [, A_lo] 128x64 and W
//              256x64, bf16, 128-byte swizzle; 4 stages of 48 KB, or 3 of
//              64 KB when split), one mbarrier per stage with transaction bytes;
//   warp 1     allocates 256 TMEM columns, one lane issues tcgen05.mma
//              (M 128, N 256, K 16) and frees a stage with tcgen05.commit;
//   warps 2-5  epilogue: tcgen05.ld of their 32-lane quadrant, one output row
//              per thread.
// Tiles are rasterised M-fastest so that the CTAs sharing a weight tile run
// together and read it from HBM once.  Every mbarrier wait is bounded; on
// timeout the kernel records an error code, stops issuing, lets its copies and
// MMAs finish, frees its TMEM and returns.
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
constexpr int kThreadsTC = 192;
constexpr uint32_t kTmemCols = 256;
// instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, N = 256, M = 128
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(TBN >> 3) << 17) |
                            ((uint32_t)(TBM >> 4) << 24);

enum { T_QKV = 0, T_RESID = 1, T_SWIGLU = 2 };

struct TcParams {
    int M, N, K;  // N: output columns (QKV, RESID) or F (SWIGLU)
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
__device__ __forceinline__ uint16_t f2bf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }
__device__ __forceinline__ float bf2f(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }

__device__ __forceinline__ void record_error(int code) { atomicCAS(&g_tc_error, 0, code); }

template <int EPI>
__device__ __forceinline__ void epilogue(const TcParams& p, uint32_t tbase, int row, int ntile) {
    const bool live = row < p.M;
    if (EPI == T_RESID) {
        const int n0 = ntile * TBN;
#pragma unroll 1
        for (int c0 = 0; c0 < TBN; c0 += 32) {
            float v[32];
            tmem_ld32(tbase + c0, v);
            if (!live) continue;
            float* xr = p.x + (size_t)row * p.N + n0 + c0;
            if (n0 + c0 + 32 <= p.N) {
#pragma unroll
                for (int j = 0; j < 32; j += 4) {
                    float4 t = *reinterpret_cast<float4*>(xr + j);
                    t.x += v[j];
                    t.y += v[j + 1];
                    t.z += v[j + 2];
                    t.w += v[j + 3];
                    *reinterpret_cast<float4*>(xr + j) = t;
                }
            } else {
                for (int j = 0; j < 32; ++j)
                    if (n0 + c0 + j < p.N) xr[j] += v[j];
            }
        }
    } else if (EPI == T_SWIGLU) {
        const int f0 = ntile * 128;
#pragma unroll 1
        for (int c0 = 0; c0 < 128; c0 += 32) {
            float g[32], u[32];
            tmem_ld32(tbase + c0, g);
            tmem_ld32(tbase + 128 + c0, u);
            if (!live) continue;
            uint16_t* ar = p.a + (size_t)row * p.N + f0 + c0;
            const size_t plane = (size_t)p.M * p.N;
            if (f0 + c0 + 32 <= p.N) {
#pragma unroll
                for (int j = 0; j < 32; j += 8) {
                    uint32_t w[4], wl[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float s0 = g[j + 2 * e] / (1.0f + expf(-g[j + 2 * e])) * u[j + 2 * e];
                        const float s1 = g[j + 2 * e + 1] / (1.0f + expf(-g[j + 2 * e + 1])) * u[j + 2 * e + 1];
                        const uint16_t h0 = f2bf(s0), h1 = f2bf(s1);
                        w[e] = (uint32_t)h0 | ((uint32_t)h1 << 16);
                        wl[e] = (uint32_t)f2bf(s0 - bf2f(h0)) | ((uint32_t)f2bf(s1 - bf2f(h1)) << 16);
                    }
                    *reinterpret_cast<uint4*>(ar + j) = make_uint4(w[0], w[1], w[2], w[3]);
                    *reinterpret_cast<uint4*>(ar + plane + j) = make_uint4(wl[0], wl[1], wl[2], wl[3]);
                }
            } else {
                for (int j = 0; j < 32; ++j)
                    if (f0 + c0 + j < p.N) {
                        const float sv = g[j] / (1.0f + expf(-g[j])) * u[j];
                        const uint16_t h = f2bf(sv);
                        ar[j] = h;
                        ar[plane + j] = f2bf(sv - bf2f(h));
                    }
            }
        }
    } else {  // T_QKV: the tile holds 256 / d whole heads
        const int n0 = ntile * TBN, d = p.d, half = d >> 1;
        const int pos = live ? p.positions[row] : 0;
#pragma unroll 1
        for (int hc = 0; hc < TBN; hc += d) {
            if (n0 + hc >= p.N) break;  // uniform across the warp
            const int h = (n0 + hc) / d;
#pragma unroll 1
            for (int i0 = 0; i0 < half; i0 += 32) {
                float v0[32], v1[32];
                tmem_ld32(tbase + hc + i0, v0);
                tmem_ld32(tbase + hc + half + i0, v1);
                if (!live) continue;
                if (h < p.Hq + p.Hkv) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        float c, s;
                        rope_cos_sin(pos, p.rope.inv_freq[i0 + j], &c, &s);
                        const float r0 = v0[j] * c - v1[j] * s, r1 = v1[j] * c + v0[j] * s;
                        v0[j] = r0;
                        v1[j] = r1;
                    }
                }
                if (h < p.Hq) {
                    float* qr = p.q + (size_t)row * p.Hq * d + (size_t)h * d + i0;
#pragma unroll
                    for (int j = 0; j < 32; j += 4) {
                        *reinterpret_cast<float4*>(qr + j) = make_float4(v0[j], v0[j + 1], v0[j + 2], v0[j + 3]);
                        *reinterpret_cast<float4*>(qr + half + j) =
                            make_float4(v1[j], v1[j + 1], v1[j + 2], v1[j + 3]);
                    }
                } else {
                    const bool is_v = h >= p.Hq + p.Hkv;
                    const int kh = h - p.Hq - (is_v ? p.Hkv : 0);
                    const int req = p.row_req[row];
                    const int page = pos / p.kv.page_tokens, t = pos - page * p.kv.page_tokens;
                    char* base = p.kv.base + p.kv.page_offsets[(int64_t)req * p.kv.max_pages + page] +
                                 (uint64_t)p.kv.layer * p.kv.layer_page_bytes;
                    uint16_t* kr = reinterpret_cast<uint16_t*>(
                        base + ((uint64_t)((is_v ? p.Hkv : 0) + kh) * p.kv.page_tokens + t) * (uint64_t)d * 2u);
#pragma unroll
                    for (int j = 0; j < 32; j += 8) {
                        uint32_t w0[4], w1[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            w0[e] = (uint32_t)f2bf(v0[j + 2 * e]) | ((uint32_t)f2bf(v0[j + 2 * e + 1]) << 16);
                            w1[e] = (uint32_t)f2bf(v1[j + 2 * e]) | ((uint32_t)f2bf(v1[j + 2 * e + 1]) << 16);
                        }
                        *reinterpret_cast<uint4*>(kr + i0 + j) = make_uint4(w0[0], w0[1], w0[2], w0[3]);
                        *reinterpret_cast<uint4*>(kr + half + i0 + j) = make_uint4(w1[0], w1[1], w1[2], w1[3]);
                    }
                }
            }
        }
    }
}

template <int EPI, int SPLIT>
__global__ void __launch_bounds__(kThreadsTC, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmAlo,
                   const __grid_constant__ CUtensorMap tmB0, const __grid_constant__ CUtensorMap tmB1, TcParams p) {
    constexpr int STAGES = Ring<SPLIT>::STAGES, STAGE_BYTES = Ring<SPLIT>::STAGE_BYTES, B_OFF = Ring<SPLIT>::B_OFF;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * TBM, ntile = blockIdx.y;
    const int nk = (p.K + TBK - 1) / TBK;
    const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + STAGES), accb = smem_u32(bars + 2 * STAGES);

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, 1);
        }
        mbar_init(accb, 1);
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
            const int y0 = (EPI == T_SWIGLU) ? ntile * 128 : ntile * TBN;
            const int y1 = (EPI == T_SWIGLU) ? ntile * 128 : ntile * TBN + 128;
            int issued = 0;
            for (int kb = 0; kb < nk; ++kb) {
                const int s = kb % STAGES;
                const uint32_t ph = (kb / STAGES) & 1;
                if (!mbar_wait(empty0 + 8 * s, ph ^ 1)) {
                    record_error(1);
                    break;
                }
                const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
                mbar_expect_tx(full0 + 8 * s, STAGE_BYTES);
                tma_load_2d(sa, &tmA, kb * TBK, m0, full0 + 8 * s);
                if (SPLIT) tma_load_2d(sa + A_BYTES, &tmAlo, kb * TBK, m0, full0 + 8 * s);
                tma_load_2d(sa + B_OFF, &tmB0, kb * TBK, y0, full0 + 8 * s);
                tma_load_2d(sa + B_OFF + B_HALF, mb1, kb * TBK, y1, full0 + 8 * s);
                ++issued;
            }
            // the copies of the last stages must land before this CTA's shared
            // memory can be released
            for (int kb = issued - STAGES < 0 ? 0 : issued - STAGES; kb < issued; ++kb)
                if (!mbar_wait(full0 + 8 * (kb % STAGES), (kb / STAGES) & 1)) record_error(4);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            for (int kb = 0; kb < nk; ++kb) {
                const int s = kb % STAGES;
                const uint32_t ph = (kb / STAGES) & 1;
                if (!mbar_wait(full0 + 8 * s, ph)) {
                    record_error(2);
                    break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t sa = smem_u32(smem + s * STAGE_BYTES);
                const uint64_t da = smem_desc(sa), db = smem_desc(sa + B_OFF);
#pragma unroll
                for (int k = 0; k < TBK / 16; ++k) {  // 32 bytes along K per instruction
                    umma_bf16(tmem, da + 2 * k, db + 2 * k, (kb | k) != 0 ? 1u : 0u);
                    if (SPLIT) umma_bf16(tmem, smem_desc(sa + A_BYTES) + 2 * k, db + 2 * k, 1u);  // + A_lo W^T
                }
                umma_commit(empty0 + 8 * s);
            }
            umma_commit(accb);  // arrives once every MMA issued above has completed
        }
        __syncwarp();
    } else {
        const int quad = warp & 3;  // TMEM lanes 32*quad .. 32*quad+31
        const int row = m0 + quad * 32 + lane;
        bool ok = mbar_wait(accb, 0);
        if (!ok) record_error(3);
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        ok = __all_sync(0xffffffffu, ok) && *(volatile int*)&g_tc_error == 0;
        if (ok) epilogue<EPI>(p, tmem + ((uint32_t)(quad * 32) << 16), row, ntile);
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
    dim3 grid((p.M + TBM - 1) / TBM, n_tiles);
    tc_gemm_kernel<EPI, SPLIT><<<grid, kThreadsTC, SMEM, st>>>(ma, malo, mb0, mb1, p);
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
