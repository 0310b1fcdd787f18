// decode.cu -- the decode-time kernels of one LLaMA-style decoder layer on
// sm_103a, plus the embedding gather, the LM head with greedy argmax and the
// seeded weight generator.
//
// Every decode projection is a weight-stationary matrix-vector product that is
// HBM bound: each bf16 weight byte is read exactly once with 128-bit streaming
// loads (ld.global.nc.L1::no_allocate), the fp32 activation rows are staged in
// shared memory in a bank-conflict-free permuted layout, each warp owns a few
// output rows and reduces its partial sums with xor shuffles.  Normalisation,
// rotary embedding, KV-cache append, SwiGLU, residual adds and the argmax are
// fused into the prologue/epilogue of the product that produces their input,
// so activations never take an extra trip through HBM.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <utility>

#include "internal.h"

namespace loip {
namespace {

constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr int kStageFloats = 16384;  // 64 KB of staged activations per block
constexpr int kMaxChunks = 256;      // pages per request in split attention (16384 positions)
#ifndef LOIP_GEMV_MIN_BLOCKS1
#define LOIP_GEMV_MIN_BLOCKS1 2  // resident blocks per SM the registers are sized for, batch tile 1
#endif
#ifndef LOIP_GEMV_JU1
#define LOIP_GEMV_JU1 4  // 128-bit loads per row and batch at batch tile 1
#endif

__device__ __forceinline__ uint4 ld_stream(const uint16_t* p) {
    uint4 r;
    asm("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
        : "l"(p));
    return r;
}
__device__ __forceinline__ float bf_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf_hi(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }
__device__ __forceinline__ float bf2f(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }
__device__ __forceinline__ uint16_t f2bf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }

// Programmatic dependent launch: let the next kernel of the stream start its
// independent prologue, and wait for the previous kernel's results.  Both are
// no-ops for a kernel launched without the attribute.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Orderable 64-bit argmax key: larger value wins; on equal values the lower
// index wins (the low word stores ~index).
__device__ __forceinline__ uint64_t argmax_key(float v, uint32_t idx) {
    uint32_t u = __float_as_uint(v);
    u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
    return ((uint64_t)u << 32) | (uint64_t)(0xffffffffu - idx);
}

__device__ __forceinline__ char* kv_row(const KvView& kv, int req, int pos, int kv_or_v, int head, int Hkv, int d) {
    int page = pos / kv.page_tokens, t = pos - page * kv.page_tokens;
    char* p = kv.base + kv.page_offsets[(int64_t)req * kv.max_pages + page] + (uint64_t)kv.layer * kv.layer_page_bytes;
    p += ((uint64_t)(kv_or_v * Hkv + head) * kv.page_tokens + t) * (uint64_t)d * 2u;
    return p;
}

// ----------------------------------------------------------------------------
// Matrix-vector family
// ----------------------------------------------------------------------------
enum { EPI_QKV = 0, EPI_RESID = 1, EPI_SWIGLU = 2, EPI_LOGITS = 3 };

struct GemvParams {
    const float* in;     // [B, K] fp32 activations
    const uint16_t* g;   // [K] gain: input is RMSNorm(in) * g when non-null
    const uint16_t* w0;  // [N, K]
    const uint16_t* w1;  // [N, K] (SwiGLU up projection)
    int B, K, N, n_units;
    float eps;
    float* out;
    float* z;
    uint64_t* keys;
    // QKV epilogue
    int Hq, Hkv, d;
    const int32_t* positions;
    const int32_t* row_req;
    KvView kv;
    RopeFreqs rope;
    int w_host;  // weights are read in place from mapped host memory: no L2 prefetch of them
    float* qk_raw;  // QK-norm models: query/key rows leave unrotated here ([B][(Hq + 2 Hkv) d])
    int pf_stride;  // block-tile kernel, > 0: before its dependency wait, block b pulls tiles
                    // b + pf_stride, b + 2 pf_stride, ... (the later waves) into L2
};

// rows handled per warp unit, by epilogue
template <int EPI>
struct UnitRows {
    static constexpr int U = EPI == EPI_RESID ? 1 : 2;
};

template <int EPI>
__device__ __forceinline__ const uint16_t* unit_row(const GemvParams& p, int unit, int r, bool& valid) {
    if (EPI == EPI_QKV) {
        int half = p.d >> 1;
        int h = unit / half, i = unit - h * half;
        valid = unit < p.n_units;
        return p.w0 + (size_t)(h * p.d + i + r * half) * p.K;
    } else if (EPI == EPI_SWIGLU) {
        valid = unit < p.n_units;
        return (r ? p.w1 : p.w0) + (size_t)unit * p.K;
    } else {
        int row = unit * UnitRows<EPI>::U + r;
        valid = row < p.N;
        return p.w0 + (size_t)row * p.K;
    }
}

// Staged-activation index of element k of row b inside a chunk.
template <int BT>
__device__ __forceinline__ int stage_index(int k, int b) {
    int j = k >> 8, lane = (k >> 3) & 31;
    if (BT == 1) {
        int half = (k >> 2) & 1, e4 = k & 3;
        return ((j * 2 + half) * 32 + lane) * 4 + e4;
    } else {
        int e = k & 7;
        return ((j * 8 + e) * BT + b) * 32 + lane;
    }
}

template <int BT, int U>
__device__ __forceinline__ void fma_block(float (&acc)[U][BT], const uint4 (&w)[U], const float* __restrict__ s,
                                          int j, int lane) {
    if (BT == 1) {
        const float4* s4 = reinterpret_cast<const float4*>(s);
        float4 ya = s4[(j * 2) * 32 + lane], yb = s4[(j * 2 + 1) * 32 + lane];
#pragma unroll
        for (int r = 0; r < U; ++r) {
            float a = acc[r][0];
            a = fmaf(bf_lo(w[r].x), ya.x, a);
            a = fmaf(bf_hi(w[r].x), ya.y, a);
            a = fmaf(bf_lo(w[r].y), ya.z, a);
            a = fmaf(bf_hi(w[r].y), ya.w, a);
            a = fmaf(bf_lo(w[r].z), yb.x, a);
            a = fmaf(bf_hi(w[r].z), yb.y, a);
            a = fmaf(bf_lo(w[r].w), yb.z, a);
            a = fmaf(bf_hi(w[r].w), yb.w, a);
            acc[r][0] = a;
        }
    } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            float wf[U];
#pragma unroll
            for (int r = 0; r < U; ++r) {
                uint32_t word = (e < 2) ? w[r].x : (e < 4) ? w[r].y : (e < 6) ? w[r].z : w[r].w;
                wf[r] = (e & 1) ? bf_hi(word) : bf_lo(word);
            }
#pragma unroll
            for (int b = 0; b < BT; ++b) {
                float y = s[((j * 8 + e) * BT + b) * 32 + lane];
#pragma unroll
                for (int r = 0; r < U; ++r) acc[r][b] = fmaf(wf[r], y, acc[r][b]);
            }
        }
    }
}

// Accumulates the unit's rows over staged chunk [kc0, kc0 + kn).  Two register
// batches of JU 128-bit loads per row alternate, so the next batch is in flight
// while the current one is consumed.
template <int BT, int U, int JU>
__device__ __forceinline__ void load_batch(uint4 (&w)[JU][U], const uint16_t* const (&rp)[U], const bool (&rv)[U],
                                           int kc0, int j0, int nj, int K, int lane) {
#pragma unroll
    for (int jj = 0; jj < JU; ++jj) {
        const int k = kc0 + (j0 + jj) * 256 + lane * 8;
        const bool ok = (j0 + jj < nj) && (k < K);
#pragma unroll
        for (int r = 0; r < U; ++r) w[jj][r] = (ok && rv[r]) ? ld_stream(rp[r] + k) : make_uint4(0, 0, 0, 0);
    }
}

// Loads per row and batch: a warp keeps about 2 x 8 x 16 bytes per lane in
// flight whatever its unit's row count.
template <int BT, int U>
struct Batch {
    static constexpr int JU = (BT == 1) ? (U == 1 ? 2 * LOIP_GEMV_JU1 : LOIP_GEMV_JU1) : (BT == 2) ? 4 : 2;
};

template <int BT, int U, int EPI>
__device__ __forceinline__ void unit_chunk(float (&acc)[U][BT], const uint16_t* const (&rp)[U], const bool (&rv)[U],
                                           const float* __restrict__ s, int kc0, int kn, int K, int lane) {
    constexpr int JU = Batch<BT, U>::JU;
    const int nj = (kn + 255) >> 8;
    uint4 wa[JU][U], wb[JU][U];
    load_batch<BT, U, JU>(wa, rp, rv, kc0, 0, nj, K, lane);
    for (int j0 = 0; j0 < nj; j0 += 2 * JU) {
        load_batch<BT, U, JU>(wb, rp, rv, kc0, j0 + JU, nj, K, lane);
#pragma unroll
        for (int jj = 0; jj < JU; ++jj)
            if (j0 + jj < nj) fma_block<BT, U>(acc, wa[jj], s, j0 + jj, lane);
        load_batch<BT, U, JU>(wa, rp, rv, kc0, j0 + 2 * JU, nj, K, lane);
#pragma unroll
        for (int jj = 0; jj < JU; ++jj)
            if (j0 + JU + jj < nj) fma_block<BT, U>(acc, wb[jj], s, j0 + JU + jj, lane);
    }
}

template <int BT, int U, int EPI>
__device__ __forceinline__ void unit_epilogue(const GemvParams& p, int unit, float (&acc)[U][BT], const float* inv,
                                              int lane, uint64_t (&best)[BT]) {
#pragma unroll
    for (int r = 0; r < U; ++r)
#pragma unroll
        for (int b = 0; b < BT; ++b) acc[r][b] = warp_sum(acc[r][b]);
    if (EPI == EPI_QKV) {
        if (unit >= p.n_units) return;
        const int half = p.d >> 1;
        const int h = unit / half, i = unit - h * half;
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            if (lane != b || b >= p.B) continue;
            float v0 = acc[0][b] * inv[b], v1 = acc[1][b] * inv[b];
            const int pos = p.positions[b];
            if (p.qk_raw && h < p.Hq + p.Hkv) {  // normalised and rotated by qk_norm_rope_kernel
                float* raw = p.qk_raw + (size_t)b * (p.Hq + 2 * p.Hkv) * p.d + (size_t)h * p.d;
                raw[i] = v0;
                raw[i + half] = v1;
                continue;
            }
            if (h < p.Hq + p.Hkv) {
                float cf, sf;
                rope_cos_sin(pos, p.rope.inv_freq[i], &cf, &sf);
                float r0 = v0 * cf - v1 * sf, r1 = v1 * cf + v0 * sf;
                v0 = r0;
                v1 = r1;
            }
            if (h < p.Hq) {
                float* q = p.out + (size_t)b * p.Hq * p.d + (size_t)h * p.d;
                q[i] = v0;
                q[i + half] = v1;
            } else {
                const int req = p.row_req ? p.row_req[b] : b;
                const bool is_v = h >= p.Hq + p.Hkv;
                const int kh = h - p.Hq - (is_v ? p.Hkv : 0);
                uint16_t* row = reinterpret_cast<uint16_t*>(kv_row(p.kv, req, pos, is_v ? 1 : 0, kh, p.Hkv, p.d));
                row[i] = f2bf(v0);
                row[i + half] = f2bf(v1);
            }
        }
    } else if (EPI == EPI_RESID) {
#pragma unroll
        for (int r = 0; r < U; ++r)
#pragma unroll
            for (int b = 0; b < BT; ++b) {
                int row = unit * U + r;
                if (lane == r * BT + b && b < p.B && row < p.N) p.out[(size_t)b * p.N + row] += acc[r][b];
            }
    } else if (EPI == EPI_SWIGLU) {
        if (unit >= p.n_units) return;
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            if (lane != b || b >= p.B) continue;
            float gt = acc[0][b] * inv[b], ut = acc[1][b] * inv[b];
            float silu = gt / (1.0f + expf(-gt));
            p.out[(size_t)b * p.N + unit] = silu * ut;
        }
    } else {  // EPI_LOGITS
#pragma unroll
        for (int r = 0; r < U; ++r) {
            int row = unit * U + r;
            if (row >= p.N) continue;
#pragma unroll
            for (int b = 0; b < BT; ++b) {
                if (b >= p.B) continue;
                float v = acc[r][b] * inv[b];
                if (p.out && lane == r * BT + b) p.out[(size_t)b * p.N + row] = v;
                uint64_t key = argmax_key(v, (uint32_t)row);
                best[b] = key > best[b] ? key : best[b];
            }
        }
    }
}

template <int BT, int EPI>
__global__ void __launch_bounds__(kThreads, BT == 1 ? LOIP_GEMV_MIN_BLOCKS1 : 2) gemv_kernel(GemvParams p) {
    constexpr int U = UnitRows<EPI>::U;
    extern __shared__ __align__(16) float s_stage[];
    __shared__ float s_red[kWarps][BT];
    __shared__ float s_inv[BT];
    __shared__ uint64_t s_keys[kWarps][BT];

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int K = p.K;
    int kc_max = (kStageFloats / BT) & ~255;
    const bool single = K <= kc_max;
    const int KC = single ? ((K + 255) & ~255) : kc_max;
    const bool norm = p.g != nullptr;

    // weights never depend on the previous kernel: start pulling this warp's
    // first rows (up to 32 KB each) into L2 before waiting for the activations
    pdl_trigger();
    {
        const int u0 = blockIdx.x * kWarps + warp;
        if (!p.w_host && lane < U && u0 < p.n_units) {
            bool v;
            const uint16_t* r = unit_row<EPI>(p, u0, lane, v);
            const uint32_t bytes = (uint32_t)min(K * 2, 32768);
            if (v) prefetch_l2(r, bytes);
        }
    }
    pdl_wait();

    float ss[BT];
#pragma unroll
    for (int b = 0; b < BT; ++b) ss[b] = 0.f;
    uint64_t best[BT];
#pragma unroll
    for (int b = 0; b < BT; ++b) best[b] = 0;

    // Stages chunk [kc0, kc0 + KC) of every activation row: 16-byte loads, four
    // per thread issued before any is consumed, so one L2 round trip covers
    // 4 x 256 x 16 bytes; zeros pad the chunk to a multiple of 256 elements.
    auto stage = [&](int kc0) {
        const int kn = min(KC, K - kc0), kpad = (kn + 255) & ~255;
        const int n4 = kpad >> 2;
        constexpr int UN = 4;
#pragma unroll
        for (int b = 0; b < BT; ++b) {
            for (int base = tid; base < n4; base += kThreads * UN) {
                float4 v[UN];
                uint2 gv[UN];
#pragma unroll
                for (int u = 0; u < UN; ++u) {
                    const int k = (base + u * kThreads) * 4;
                    const bool ok = k < kn && b < p.B;
                    v[u] = ok ? *reinterpret_cast<const float4*>(p.in + (size_t)b * K + kc0 + k)
                              : make_float4(0.f, 0.f, 0.f, 0.f);
                    gv[u] = (ok && norm) ? *reinterpret_cast<const uint2*>(p.g + kc0 + k) : make_uint2(0, 0);
                }
#pragma unroll
                for (int u = 0; u < UN; ++u) {
                    const int k = (base + u * kThreads) * 4;
                    if (k >= kpad) continue;
                    float4 w = v[u];
                    if (norm) {
                        ss[b] = fmaf(w.x, w.x, ss[b]);
                        ss[b] = fmaf(w.y, w.y, ss[b]);
                        ss[b] = fmaf(w.z, w.z, ss[b]);
                        ss[b] = fmaf(w.w, w.w, ss[b]);
                        w.x *= bf_lo(gv[u].x);
                        w.y *= bf_hi(gv[u].x);
                        w.z *= bf_lo(gv[u].y);
                        w.w *= bf_hi(gv[u].y);
                    }
                    if (BT == 1) {
                        *reinterpret_cast<float4*>(&s_stage[stage_index<1>(k, 0)]) = w;
                    } else {
                        s_stage[stage_index<BT>(k, b)] = w.x;
                        s_stage[stage_index<BT>(k + 1, b)] = w.y;
                        s_stage[stage_index<BT>(k + 2, b)] = w.z;
                        s_stage[stage_index<BT>(k + 3, b)] = w.w;
                    }
                }
            }
        }
    };
    auto finish_norm = [&]() {
        if (norm) {
#pragma unroll
            for (int b = 0; b < BT; ++b) {
                float t = warp_sum(ss[b]);
                if (lane == 0) s_red[warp][b] = t;
            }
            __syncthreads();
            if (tid < BT) {
                float t = 0.f;
                for (int w = 0; w < kWarps; ++w) t += s_red[w][tid];
                s_inv[tid] = 1.0f / sqrtf(t / (float)K + p.eps);
            }
        } else if (tid < BT) {
            s_inv[tid] = 1.0f;
        }
        __syncthreads();
    };

    if (single) {
        stage(0);
        __syncthreads();
        finish_norm();
        float inv[BT];
#pragma unroll
        for (int b = 0; b < BT; ++b) inv[b] = s_inv[b];
        for (int unit = blockIdx.x * kWarps + warp; unit < p.n_units; unit += gridDim.x * kWarps) {
            const uint16_t* rp[U];
            bool rv[U];
#pragma unroll
            for (int r = 0; r < U; ++r) rp[r] = unit_row<EPI>(p, unit, r, rv[r]);
            float acc[U][BT];
#pragma unroll
            for (int r = 0; r < U; ++r)
#pragma unroll
                for (int b = 0; b < BT; ++b) acc[r][b] = 0.f;
            unit_chunk<BT, U, EPI>(acc, rp, rv, s_stage, 0, K, K, lane);
            unit_epilogue<BT, U, EPI>(p, unit, acc, inv, lane, best);
        }
    } else {
        const int unit = blockIdx.x * kWarps + warp;
        const uint16_t* rp[U];
        bool rv[U];
#pragma unroll
        for (int r = 0; r < U; ++r) rp[r] = unit_row<EPI>(p, unit, r, rv[r]);
        float acc[U][BT];
#pragma unroll
        for (int r = 0; r < U; ++r)
#pragma unroll
            for (int b = 0; b < BT; ++b) acc[r][b] = 0.f;
        for (int kc0 = 0; kc0 < K; kc0 += KC) {
            __syncthreads();
            stage(kc0);
            __syncthreads();
            unit_chunk<BT, U, EPI>(acc, rp, rv, s_stage, kc0, min(KC, K - kc0), K, lane);
        }
        finish_norm();
        float inv[BT];
#pragma unroll
        for (int b = 0; b < BT; ++b) inv[b] = s_inv[b];
        unit_epilogue<BT, U, EPI>(p, unit, acc, inv, lane, best);
    }

    if (EPI == EPI_LOGITS) {
        if (lane == 0)
#pragma unroll
            for (int b = 0; b < BT; ++b) s_keys[warp][b] = best[b];
        __syncthreads();
        if (tid < BT) {
            uint64_t k = 0;
            for (int w = 0; w < kWarps; ++w) k = s_keys[w][tid] > k ? s_keys[w][tid] : k;
            p.keys[(size_t)blockIdx.x * BT + tid] = k;
        }
        // final hidden z = RMSNorm(x) * g, written once
        if (blockIdx.x == 0 && p.z) {
            for (int b = 0; b < p.B; ++b)
                for (int k = tid; k < K; k += kThreads)
                    p.z[(size_t)b * K + k] = p.in[(size_t)b * K + k] * s_inv[b] * bf2f(p.g[k]);
        }
    }
}

// ----------------------------------------------------------------------------
// Batch-1 block-tile GEMV.  A block owns kTileRows weight rows; its warps split
// K, so every 128-bit load of the tile is issued within one or two batches per
// warp (double-buffered), and the activation slice a warp needs comes straight
// from L1/L2 (no staging barrier).  Partial sums are reduced in a fixed order
// (lanes, then warps) so results do not depend on scheduling.  Row units as in
// the persistent kernel: QKV and SwiGLU tiles hold 4 row pairs.
// ----------------------------------------------------------------------------
constexpr int kTileWarps = 8;
constexpr int kTileRows = 8;

template <int EPI>
__device__ __forceinline__ const uint16_t* tile_row(const GemvParams& p, int tile, int r, bool& valid) {
    if (EPI == EPI_QKV) {
        const int half = p.d >> 1;
        const int pair = tile * (kTileRows / 2) + (r & 3);
        const int h = pair / half, i = pair - h * half;
        valid = pair < p.n_units;
        return p.w0 + (size_t)(h * p.d + i + (r >> 2) * half) * p.K;
    } else if (EPI == EPI_SWIGLU) {
        const int j = tile * (kTileRows / 2) + (r & 3);
        valid = j < p.n_units;
        return ((r >> 2) ? p.w1 : p.w0) + (size_t)j * p.K;
    } else {
        const int row = tile * kTileRows + r;
        valid = row < p.N;
        return p.w0 + (size_t)row * p.K;
    }
}

__device__ __forceinline__ void tile_load(uint4 (&w)[kTileRows], const uint16_t* const (&rp)[kTileRows],
                                          const bool (&rv)[kTileRows], int j, int j_end, int K, int lane) {
    const int k = j * 256 + lane * 8;
    const bool ok = j < j_end && k < K;
#pragma unroll
    for (int r = 0; r < kTileRows; ++r) w[r] = (ok && rv[r]) ? ld_stream(rp[r] + k) : make_uint4(0, 0, 0, 0);
}

// Issues the first batch of tile `tile`'s weight loads into w (this warp's
// first 256-column slice of every row).
template <int EPI>
__device__ __forceinline__ void tile_first_load(const GemvParams& p, int tile, uint4 (&w)[kTileRows]) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nj = (p.K + 255) >> 8, njw = (nj + kTileWarps - 1) / kTileWarps;
    const int j_begin = warp * njw, j_end = min(nj, j_begin + njw);
    const uint16_t* rp[kTileRows];
    bool rv[kTileRows];
#pragma unroll
    for (int r = 0; r < kTileRows; ++r) rp[r] = tile_row<EPI>(p, tile, r, rv[r]);
    tile_load(w, rp, rv, j_begin, j_end, p.K, lane);
}

struct TileShared {
    float part[kTileWarps][kTileRows];
    float ss[kTileWarps];
    float val[kTileRows];
    float inv;
};

// Activation loads.  CG: through L2 only -- the persistent layer-run kernel
// rewrites activations between its phases and L1 is not coherent across SMs.
template <bool CG>
__device__ __forceinline__ float4 ld_act4(const float* p) {
    if (CG) return __ldcg(reinterpret_cast<const float4*>(p));
    return *reinterpret_cast<const float4*>(p);
}
template <bool CG>
__device__ __forceinline__ float ld_act(const float* p) {
    return CG ? __ldcg(p) : *p;
}

// One tile of the batch-1 block-tile GEMV.  wa holds the first batch of the
// tile's loads (tile_first_load).  When next >= 0, the first batch of tile
// `next` is issued into wa as soon as this tile's loads are consumed, so its
// weights stream during this tile's reduction and epilogue.
template <int EPI, bool CG, bool STAGED = false>
__device__ __forceinline__ void tile_gemv(const GemvParams& p, int tile, int next, uint4 (&wa)[kTileRows],
                                          TileShared& sm, const float* sx = nullptr, float inv_staged = 1.f) {
    constexpr int R = kTileRows;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int K = p.K;
    const int nj = (K + 255) >> 8;
    const int njw = (nj + kTileWarps - 1) / kTileWarps;
    const int j_begin = warp * njw, j_end = min(nj, j_begin + njw);
    const bool norm = p.g != nullptr;
    const uint16_t* rp[R];
    bool rv[R];
#pragma unroll
    for (int r = 0; r < R; ++r) rp[r] = tile_row<EPI>(p, tile, r, rv[r]);

    uint4 wb[R];
    float acc[R];
#pragma unroll
    for (int r = 0; r < R; ++r) acc[r] = 0.f;
    float ss = 0.f;
    auto consume = [&](const uint4 (&w)[R], int j) {
        const int k = j * 256 + lane * 8;
        if (j >= j_end || k >= K) return;
        const float4 xa = STAGED ? *reinterpret_cast<const float4*>(sx + k) : ld_act4<CG>(p.in + k);
        const float4 xb = STAGED ? *reinterpret_cast<const float4*>(sx + k + 4) : ld_act4<CG>(p.in + k + 4);
        float xv[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
        if (norm && !STAGED) {  // staged inputs already carry the gain
            const uint4 gv = *reinterpret_cast<const uint4*>(p.g + k);
            const float gf[8] = {bf_lo(gv.x), bf_hi(gv.x), bf_lo(gv.y), bf_hi(gv.y),
                                 bf_lo(gv.z), bf_hi(gv.z), bf_lo(gv.w), bf_hi(gv.w)};
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                ss = fmaf(xv[e], xv[e], ss);
                xv[e] *= gf[e];
            }
        }
#pragma unroll
        for (int r = 0; r < R; ++r) {
            float a = acc[r];
            a = fmaf(bf_lo(w[r].x), xv[0], a);
            a = fmaf(bf_hi(w[r].x), xv[1], a);
            a = fmaf(bf_lo(w[r].y), xv[2], a);
            a = fmaf(bf_hi(w[r].y), xv[3], a);
            a = fmaf(bf_lo(w[r].z), xv[4], a);
            a = fmaf(bf_hi(w[r].z), xv[5], a);
            a = fmaf(bf_lo(w[r].w), xv[6], a);
            a = fmaf(bf_hi(w[r].w), xv[7], a);
            acc[r] = a;
        }
    };
    for (int j = j_begin; j < j_end; j += 2) {
        tile_load(wb, rp, rv, j + 1, j_end, K, lane);
        consume(wa, j);
        tile_load(wa, rp, rv, j + 2, j_end, K, lane);
        consume(wb, j + 1);
    }
    if (next >= 0) tile_first_load<EPI>(p, next, wa);
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const float v = warp_sum(acc[r]);
        if (lane == 0) sm.part[warp][r] = v;
    }
    if (norm && !STAGED) {
        const float v = warp_sum(ss);
        if (lane == 0) sm.ss[warp] = v;
    }
    __syncthreads();
    if (tid < R) {
        float t = 0.f;
        for (int w = 0; w < kTileWarps; ++w) t += sm.part[w][tid];
        sm.val[tid] = t;
    }
    if (!STAGED && tid == 32) {
        float t = 0.f;
        if (norm)
            for (int w = 0; w < kTileWarps; ++w) t += sm.ss[w];
        sm.inv = norm ? 1.0f / sqrtf(t / (float)K + p.eps) : 1.0f;
    }
    __syncthreads();
    const float inv = STAGED ? inv_staged : sm.inv;
    if (EPI == EPI_QKV) {
        if (tid < R / 2) {
            const int half = p.d >> 1;
            const int pair = tile * (R / 2) + tid;
            if (pair < p.n_units) {
                const int h = pair / half, i = pair - h * half;
                float v0 = sm.val[tid] * inv, v1 = sm.val[tid + R / 2] * inv;
                const int pos = p.positions[0];
                const bool raw = p.qk_raw && h < p.Hq + p.Hkv;  // normalised and rotated by qk_norm_rope_kernel
                if (raw) {
                    p.qk_raw[(size_t)h * p.d + i] = v0;
                    p.qk_raw[(size_t)h * p.d + i + half] = v1;
                } else if (h < p.Hq + p.Hkv) {
                    float cf, sf;
                    rope_cos_sin(pos, p.rope.inv_freq[i], &cf, &sf);
                    const float r0 = v0 * cf - v1 * sf, r1 = v1 * cf + v0 * sf;
                    v0 = r0;
                    v1 = r1;
                }
                if (raw) {
                } else if (h < p.Hq) {
                    float* q = p.out + (size_t)h * p.d;
                    q[i] = v0;
                    q[i + half] = v1;
                } else {
                    const int req = p.row_req ? p.row_req[0] : 0;
                    const bool is_v = h >= p.Hq + p.Hkv;
                    const int kh = h - p.Hq - (is_v ? p.Hkv : 0);
                    uint16_t* row = reinterpret_cast<uint16_t*>(kv_row(p.kv, req, pos, is_v ? 1 : 0, kh, p.Hkv, p.d));
                    row[i] = f2bf(v0);
                    row[i + half] = f2bf(v1);
                }
            }
        }
    } else if (EPI == EPI_SWIGLU) {
        if (tid < R / 2) {
            const int j = tile * (R / 2) + tid;
            if (j < p.n_units) {
                const float gt = sm.val[tid] * inv, ut = sm.val[tid + R / 2] * inv;
                p.out[j] = gt / (1.0f + expf(-gt)) * ut;
            }
        }
    } else if (EPI == EPI_RESID) {
        if (tid < R) {
            const int row = tile * R + tid;
            if (row < p.N) p.out[row] = ld_act<CG>(p.out + row) + sm.val[tid];
        }
    } else {  // EPI_LOGITS
        if (tid < R) {
            const int row = tile * R + tid;
            if (row < p.N && p.out) p.out[row] = sm.val[tid] * inv;
        }
        if (tid == 0) {
            uint64_t best = 0;
            for (int r = 0; r < R; ++r) {
                const int row = tile * R + r;
                if (row < p.N) {
                    const uint64_t key = argmax_key(sm.val[r] * inv, (uint32_t)row);
                    best = key > best ? key : best;
                }
            }
            p.keys[tile] = best;
        }
        if (tile == 0 && p.z)
            for (int k = tid; k < K; k += kTileWarps * 32) p.z[k] = p.in[k] * inv * bf2f(p.g[k]);
    }
    __syncthreads();  // the shared partials are reused by the block's next tile
}

// L2 prefetch of the weight rows of one tile (lanes 0..7 of the calling warp),
// in pieces of at most 32 KB.
template <int EPI>
__device__ __forceinline__ void prefetch_tile(const GemvParams& p, int tile, int lane) {
    if (lane < kTileRows) {
        bool v;
        const uint16_t* r = tile_row<EPI>(p, tile, lane, v);
        if (v) {
            const uint32_t bytes = (uint32_t)p.K * 2u;  // a multiple of 16 (K % 8 == 0)
            for (uint32_t off = 0; off < bytes; off += 32768u)
                prefetch_l2(reinterpret_cast<const char*>(r) + off, min(32768u, bytes - off));
        }
    }
}

template <int EPI>
__global__ void __launch_bounds__(kTileWarps * 32, 2) gemv_tile_kernel(GemvParams p) {
    __shared__ TileShared sm;
    pdl_trigger();
    uint4 wa[kTileRows];
    tile_first_load<EPI>(p, blockIdx.x, wa);  // weights do not depend on the previous kernel
    if (p.pf_stride > 0 && threadIdx.x < 32)
        for (int t = blockIdx.x + p.pf_stride; t < (int)gridDim.x; t += p.pf_stride)
            prefetch_tile<EPI>(p, t, threadIdx.x);
    pdl_wait();
    tile_gemv<EPI, false>(p, blockIdx.x, -1, wa, sm);
}

__global__ void argmax_reduce_kernel(const uint64_t* keys, int nblocks, int BT, int B, int32_t* tokens) {
    __shared__ uint64_t s[256];
    pdl_trigger();
    pdl_wait();
    const int b = blockIdx.x;
    uint64_t k = 0;
    for (int i = threadIdx.x; i < nblocks; i += blockDim.x) {
        uint64_t v = keys[(size_t)i * BT + b];
        k = v > k ? v : k;
    }
    s[threadIdx.x] = k;
    __syncthreads();
    for (int o = blockDim.x / 2; o; o >>= 1) {
        if (threadIdx.x < o) s[threadIdx.x] = s[threadIdx.x + o] > s[threadIdx.x] ? s[threadIdx.x + o] : s[threadIdx.x];
        __syncthreads();
    }
    if (threadIdx.x == 0 && b < B) tokens[b] = (int32_t)(0xffffffffu - (uint32_t)(s[0] & 0xffffffffu));
}

// Launch with programmatic stream serialisation when `pdl` (the previous
// operation on the stream is a kernel of the same chain).
template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, bool pdl,
                     Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = pdl ? at : nullptr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

template <int EPI>
cudaError_t launch_gemv(GemvParams& p, cudaStream_t st, bool pdl, int* nblocks_out = nullptr) {
    // Batch 1: matrices with few rows (QKV, O-proj, down) keep too few units per
    // warp for the persistent kernel to ramp up; the block-tile kernel issues a
    // whole tile at once.  Row-rich ones (gate/up, LM head) stream better
    // persistent, and so does a QKV of more than 8192 rows (13B: 15360, two or
    // more RoPE pairs per warp), whose tiles would take six waves.  Weights in
    // mapped host memory always go to the persistent kernel: over the host link
    // a tile's serial chunk loads along a long row (down, K = 28672) ran at
    // 183 GB/s against the link's 211, which the persistent kernel reaches.
    const int rows = (EPI == EPI_SWIGLU) ? 2 * p.n_units : p.N;
    if (p.B == 1 && !p.w_host && rows <= (EPI == EPI_QKV ? 8192 : 16384)) {
        const int per_tile = (EPI == EPI_QKV || EPI == EPI_SWIGLU) ? kTileRows / 2 : kTileRows;
        const int units = (EPI == EPI_QKV || EPI == EPI_SWIGLU) ? p.n_units : p.N;
        const int tiles = (units + per_tile - 1) / per_tile;
        if (nblocks_out) *nblocks_out = tiles;
        return launch_k(gemv_tile_kernel<EPI>, dim3(tiles), dim3(kTileWarps * 32), 0, st, pdl, p);
    }
    int BT = p.B <= 1 ? 1 : p.B <= 2 ? 2 : p.B <= 4 ? 4 : 8;
    int kc_max = (kStageFloats / BT) & ~255;
    bool single = p.K <= kc_max;
    int KC = single ? ((p.K + 255) & ~255) : kc_max;
    size_t smem = (size_t)KC * BT * sizeof(float);
    int blocks = (p.n_units + kWarps - 1) / kWarps;
    static bool attr_set = false;
    if (!attr_set) {  // before any occupancy query: the stage is above the 48 KB default
        int bytes = kStageFloats * (int)sizeof(float);
        cudaFuncSetAttribute(gemv_kernel<1, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
        cudaFuncSetAttribute(gemv_kernel<2, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
        cudaFuncSetAttribute(gemv_kernel<4, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
        cudaFuncSetAttribute(gemv_kernel<8, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
        attr_set = true;
    }
    if (single) {
        // resident blocks per SM for this stage size (cached per batch tile and size)
        static int cache_bt[16], cache_smem[16], cache_val[16], cache_n = 0;
        static int sms = 0;
        int per_sm = 0;
        for (int i = 0; i < cache_n; ++i)
            if (cache_bt[i] == BT && cache_smem[i] == (int)smem) per_sm = cache_val[i];
        if (per_sm == 0) {
            int dev;
            cudaGetDevice(&dev);
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            int v = 0;
            switch (BT) {
                case 1: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, gemv_kernel<1, EPI>, kThreads, smem); break;
                case 2: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, gemv_kernel<2, EPI>, kThreads, smem); break;
                case 4: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, gemv_kernel<4, EPI>, kThreads, smem); break;
                default: cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, gemv_kernel<8, EPI>, kThreads, smem); break;
            }
            per_sm = v < 1 ? 1 : v;
            if (cache_n < 16) {
                cache_bt[cache_n] = BT;
                cache_smem[cache_n] = (int)smem;
                cache_val[cache_n] = per_sm;
                ++cache_n;
            }
        }
        int cap = per_sm * sms;
        if (blocks > cap) blocks = cap;
    }
    if (blocks < 1) blocks = 1;
    if (nblocks_out) *nblocks_out = blocks;

    switch (BT) {
        case 1: return launch_k(gemv_kernel<1, EPI>, dim3(blocks), dim3(kThreads), smem, st, pdl, p);
        case 2: return launch_k(gemv_kernel<2, EPI>, dim3(blocks), dim3(kThreads), smem, st, pdl, p);
        case 4: return launch_k(gemv_kernel<4, EPI>, dim3(blocks), dim3(kThreads), smem, st, pdl, p);
        default: return launch_k(gemv_kernel<8, EPI>, dim3(blocks), dim3(kThreads), smem, st, pdl, p);
    }
}

// ----------------------------------------------------------------------------
// Attention
// ----------------------------------------------------------------------------
struct AttnParams {
    const float* q;  // [B, Hq*d]
    KvView kv;
    const int32_t* ctx_lens;
    const int32_t* positions;  // used when ctx_lens is null: ctx = position + 1
    const int32_t* row_req;
    int B, Hq, Hkv, max_chunks;
    float scale;
    float* scratch;  // split: [B][Hq][max_chunks][d + 2] partial states, then int counters [B][Hq]
    int* counters;
    void* o;         // [B, Hq*d] fp32, or (o_split) two bf16 planes [2][B][Hq*d]
    int o_split;
    int split;  // kAttnSingle, kAttnSplit or kAttnWide
};
// single: one 64-thread block per (row, kv head) over every page; split: one
// 64-thread block per page, partial states in global scratch, combined by the
// last block to finish; wide: split with a 256-thread block per page
enum { kAttnSingle = 0, kAttnSplit = 1, kAttnWide = 2 };

// Attention output element idx: fp32, or (o_split, the prefill's tensor-core
// operand) the pair hi = bf16(v) in the first plane and lo = bf16(v - hi) in the
// second, B * Hq * d elements further on; hi + lo carries v to ~2^-17 relative.
template <int D>
__device__ __forceinline__ void store_o(const AttnParams& p, size_t idx, float v) {
    if (p.o_split) {
        uint16_t* o16 = reinterpret_cast<uint16_t*>(p.o);
        const uint16_t hi = f2bf(v);
        o16[idx] = hi;
        o16[idx + (size_t)p.B * p.Hq * D] = f2bf(v - bf2f(hi));
    } else {
        reinterpret_cast<float*>(p.o)[idx] = v;
    }
}

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(smem)),
                 "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}

template <int G, int D>
struct AttnSmem {
    alignas(16) uint16_t sK[64 * D];
    alignas(16) uint16_t sV[64 * D];
    alignas(16) float sq[G][D];
    float s_m[G], s_l[G];
    float s_o[G][D];
    int s_last;
};

// Barrier among the 64 threads of one attention group (barrier 0 with 64
// threads is the whole block of the standalone kernel; the layer-run kernel
// gives each warp pair a barrier of its own).
__device__ __forceinline__ void group_sync(int bar_id) { asm volatile("bar.sync %0, 64;" ::"r"(bar_id) : "memory"); }

// Attention of one (request row, kv head) over pages [pg0, pg1) by a group of
// two warps (tid 0..63).  The page's keys and values (64 positions x d, bf16)
// are staged in shared memory with asynchronous 16-byte copies, all in flight
// together; key rows are stored with their 16-byte chunks rotated by the row
// index so that one-row-per-lane reads hit distinct banks.  Each warp scores 32
// positions for the G query heads of the kv head (online softmax), then
// accumulates the values with the weights broadcast by shuffles; the two warps
// merge through shared memory.  Split mode (one group per page, `chunk` = page):
// the partial state goes to scratch and the last group of this (row, kv head)
// to finish combines every page's state.  CG: activations and partial states
// are read through L2 only (the layer-run kernel reuses their addresses).
template <int G, int D, bool CG>
__device__ __forceinline__ void attn_group(const AttnParams& p, int row, int kvh, int chunk, AttnSmem<G, D>& sm,
                                           int tid, int bar_id) {
    constexpr int DPL = D / 32;  // dims per lane in the PV product
    constexpr int CH = D / 8;    // 16-byte chunks per row
    const int lane = tid & 31, warp = tid >> 5;
    const int ctx = p.ctx_lens ? p.ctx_lens[row] : p.positions[row] + 1;
    const int P = p.kv.page_tokens;  // 64
    const int npages = (ctx + P - 1) / P;
    int pg0, pg1;
    if (p.split == kAttnSplit) {
        pg0 = chunk;
        pg1 = pg0 + 1;
        if (pg0 >= npages) return;
    } else {
        pg0 = 0;
        pg1 = npages;
    }
    const int req = p.row_req ? p.row_req[row] : row;
    {
        const float* qs = p.q + (size_t)row * p.Hq * D + (size_t)kvh * G * D;
        constexpr int NQ = G * D / 4 / 64;  // float4 per thread (G * D is a multiple of 256)
        float4 qv[NQ > 0 ? NQ : 1];
#pragma unroll
        for (int u = 0; u < NQ; ++u) qv[u] = ld_act4<CG>(qs + 4 * (tid + u * 64));
#pragma unroll
        for (int u = 0; u < NQ; ++u) reinterpret_cast<float4*>(&sm.sq[0][0])[tid + u * 64] = qv[u];
        if (NQ == 0 && tid < G * D / 4) reinterpret_cast<float4*>(&sm.sq[0][0])[tid] = ld_act4<CG>(qs + 4 * tid);
    }

    float m[G], l[G], o[G][DPL];
#pragma unroll
    for (int g = 0; g < G; ++g) {
        m[g] = -INFINITY;
        l[g] = 0.f;
#pragma unroll
        for (int c = 0; c < DPL; ++c) o[g][c] = 0.f;
    }
    const int Hkv = p.Hkv;
    for (int pg = pg0; pg < pg1; ++pg) {
        const int nvalid = min(P, ctx - pg * P);
        const char* page = p.kv.base + p.kv.page_offsets[(int64_t)req * p.kv.max_pages + pg] +
                           (uint64_t)p.kv.layer * p.kv.layer_page_bytes;
        const uint16_t* Kh = reinterpret_cast<const uint16_t*>(page) + (size_t)kvh * P * D;
        const uint16_t* Vh = reinterpret_cast<const uint16_t*>(page) + ((size_t)Hkv + kvh) * P * D;
        if (pg != pg0) group_sync(bar_id);  // the previous page's rows are no longer read
        for (int i = tid; i < 64 * CH; i += 64) {
            const int t = i / CH, c = i - t * CH;
            if (t < nvalid) {
                cp_async16(&sm.sK[(t * CH + ((c + t) & (CH - 1))) * 8], Kh + (size_t)t * D + c * 8);
                cp_async16(&sm.sV[(t * CH + c) * 8], Vh + (size_t)t * D + c * 8);
            } else {
                *reinterpret_cast<uint4*>(&sm.sV[(t * CH + c) * 8]) = make_uint4(0, 0, 0, 0);
            }
        }
        cp_async_wait_all();
        group_sync(bar_id);
        {
            const int tl = warp * 32 + lane;
            const bool valid = tl < nvalid;
            float sc[G];
#pragma unroll
            for (int g = 0; g < G; ++g) sc[g] = 0.f;
            if (valid) {
#pragma unroll 4
                for (int u = 0; u < CH; ++u) {
                    const uint4 kk = *reinterpret_cast<const uint4*>(&sm.sK[(tl * CH + ((u + tl) & (CH - 1))) * 8]);
                    const float kf[8] = {bf_lo(kk.x), bf_hi(kk.x), bf_lo(kk.y), bf_hi(kk.y),
                                         bf_lo(kk.z), bf_hi(kk.z), bf_lo(kk.w), bf_hi(kk.w)};
#pragma unroll
                    for (int g = 0; g < G; ++g) {
                        const float4 qa = *reinterpret_cast<const float4*>(&sm.sq[g][u * 8]);
                        const float4 qb = *reinterpret_cast<const float4*>(&sm.sq[g][u * 8 + 4]);
                        float a = sc[g];
                        a = fmaf(qa.x, kf[0], a);
                        a = fmaf(qa.y, kf[1], a);
                        a = fmaf(qa.z, kf[2], a);
                        a = fmaf(qa.w, kf[3], a);
                        a = fmaf(qb.x, kf[4], a);
                        a = fmaf(qb.y, kf[5], a);
                        a = fmaf(qb.z, kf[6], a);
                        a = fmaf(qb.w, kf[7], a);
                        sc[g] = a;
                    }
                }
            }
            float pe[G];
#pragma unroll
            for (int g = 0; g < G; ++g) {
                float sv = valid ? sc[g] * p.scale : -INFINITY;
                float mx = warp_max(sv);
                float mn = fmaxf(m[g], mx);
                float corr = (m[g] == -INFINITY) ? 0.f : expf(m[g] - mn);
                pe[g] = valid ? expf(sv - mn) : 0.f;
                l[g] = l[g] * corr + warp_sum(pe[g]);
#pragma unroll
                for (int c = 0; c < DPL; ++c) o[g][c] *= corr;
                m[g] = mn;
            }
            const int nt = min(32, nvalid - warp * 32);
            for (int u = 0; u < nt; ++u) {
                const uint16_t* vr = &sm.sV[(warp * 32 + u) * D + lane * DPL];
                float vf[DPL];
                if constexpr (DPL == 4) {
                    const uint2 vv = *reinterpret_cast<const uint2*>(vr);
                    vf[0] = bf_lo(vv.x);
                    vf[1] = bf_hi(vv.x);
                    vf[2] = bf_lo(vv.y);
                    vf[3] = bf_hi(vv.y);
                } else {
                    static_assert(DPL == 2, "head_dim 64 or 128");
                    const uint32_t vv = *reinterpret_cast<const uint32_t*>(vr);
                    vf[0] = bf_lo(vv);
                    vf[1] = bf_hi(vv);
                }
#pragma unroll
                for (int g = 0; g < G; ++g) {
                    const float pg_ = __shfl_sync(0xffffffffu, pe[g], u);
#pragma unroll
                    for (int c = 0; c < DPL; ++c) o[g][c] = fmaf(pg_, vf[c], o[g][c]);
                }
            }
        }
    }
    // merge the two warps
    if (warp == 1) {
#pragma unroll
        for (int g = 0; g < G; ++g) {
            if (lane == 0) {
                sm.s_m[g] = m[g];
                sm.s_l[g] = l[g];
            }
#pragma unroll
            for (int c = 0; c < DPL; ++c) sm.s_o[g][lane * DPL + c] = o[g][c];
        }
    }
    group_sync(bar_id);
    if (warp == 0) {
#pragma unroll
        for (int g = 0; g < G; ++g) {
            float m1 = sm.s_m[g], l1 = sm.s_l[g];
            float mn = fmaxf(m[g], m1);
            float c0 = (m[g] == -INFINITY) ? 0.f : expf(m[g] - mn);
            float c1 = (m1 == -INFINITY) ? 0.f : expf(m1 - mn);
            float lt = l[g] * c0 + l1 * c1;
            const int h = kvh * G + g;
            if (p.split == kAttnSplit) {
                float* part = p.scratch + (((size_t)row * p.Hq + h) * p.max_chunks + chunk) * (D + 2);
#pragma unroll
                for (int c = 0; c < DPL; ++c) part[lane * DPL + c] = o[g][c] * c0 + sm.s_o[g][lane * DPL + c] * c1;
                if (lane == 0) {
                    part[D] = mn;
                    part[D + 1] = lt;
                }
            } else {
                float invl = lt > 0.f ? 1.0f / lt : 0.f;
#pragma unroll
                for (int c = 0; c < DPL; ++c) {
                    float v = (o[g][c] * c0 + sm.s_o[g][lane * DPL + c] * c1) * invl;
                    size_t idx = (size_t)row * p.Hq * D + (size_t)h * D + lane * DPL + c;
                    store_o<D>(p, idx, v);
                }
            }
        }
    }
    if (p.split != kAttnSplit) return;
    // The last group of this (row, kv head) to finish combines every page's
    // state: exp-weighted sum of the partial outputs over the summed weights.
    __threadfence();
    group_sync(bar_id);
    if (tid == 0) {
        int* cnt = p.counters + (size_t)row * p.Hq + kvh;
        const int ticket = atomicAdd(cnt, 1);
        sm.s_last = ticket == npages - 1;
        if (sm.s_last) atomicExch(cnt, 0);  // every group has arrived: reset for the next launch
    }
    group_sync(bar_id);
    if (!sm.s_last) return;
    __threadfence();
    const float* base = p.scratch + ((size_t)row * p.Hq + (size_t)kvh * G) * p.max_chunks * (D + 2);
    const size_t hstride = (size_t)p.max_chunks * (D + 2);
    // the staging buffers are dead: combine weights and denominators reuse them
    static_assert(G * kMaxChunks * sizeof(float) <= sizeof(sm.sK), "combine weights fit the key stage");
    float(*s_w)[kMaxChunks] = reinterpret_cast<float(*)[kMaxChunks]>(&sm.sK[0]);
    float(*s_lw)[kMaxChunks] = reinterpret_cast<float(*)[kMaxChunks]>(&sm.sV[0]);
    // (m, l) of every (head, page) in one round trip; weights reduced in shared memory
    for (int i = tid; i < G * npages; i += 64) {
        const int g = i / npages, c = i - g * npages;
        const float* pc = base + g * hstride + (size_t)c * (D + 2);
        s_w[g][c] = ld_act<CG>(pc + D);
        s_lw[g][c] = ld_act<CG>(pc + D + 1);
    }
    group_sync(bar_id);
    for (int g = warp; g < G; g += 2) {
        float mx = -INFINITY;
        for (int c = lane; c < npages; c += 32) mx = fmaxf(mx, s_w[g][c]);
        mx = warp_max(mx);
        float lsum = 0.f;
        for (int c = lane; c < npages; c += 32) {
            const float w = (s_w[g][c] == -INFINITY) ? 0.f : expf(s_w[g][c] - mx);
            s_w[g][c] = w;
            lsum = fmaf(s_lw[g][c], w, lsum);
        }
        lsum = warp_sum(lsum);
        const float inv = lsum > 0.f ? 1.0f / lsum : 0.f;
        for (int c = lane; c < npages; c += 32) s_w[g][c] *= inv;
    }
    group_sync(bar_id);
    // chunks outer, this thread's outputs inner: 4 x NOUT loads in flight
    constexpr int NOUT = G * D / 64;
    float acc[NOUT];
#pragma unroll
    for (int k = 0; k < NOUT; ++k) acc[k] = 0.f;
    for (int c0 = 0; c0 < npages; c0 += 4) {
        float v[4][NOUT];
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int k = 0; k < NOUT; ++k) {
                const int e = tid + 64 * k, g = e / D, j = e - g * D;
                v[u][k] = (c0 + u < npages) ? ld_act<CG>(base + g * hstride + (size_t)(c0 + u) * (D + 2) + j) : 0.f;
            }
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int k = 0; k < NOUT; ++k) {
                const int g = (tid + 64 * k) / D;
                if (c0 + u < npages) acc[k] = fmaf(v[u][k], s_w[g][c0 + u], acc[k]);
            }
    }
#pragma unroll
    for (int k = 0; k < NOUT; ++k) {
        const int e = tid + 64 * k, g = e / D, j = e - g * D;
        const size_t idx = (size_t)row * p.Hq * D + (size_t)(kvh * G + g) * D + j;
        store_o<D>(p, idx, acc[k]);
    }
}

// One block of two warps per (request row, kv head, page) in split mode, or per
// (row, kv head) looping over the pages otherwise.
template <int G, int D>
__global__ void __launch_bounds__(64) attn_kernel(AttnParams p) {
    __shared__ AttnSmem<G, D> sm;
    pdl_trigger();
    pdl_wait();
    attn_group<G, D, false>(p, blockIdx.z, blockIdx.y, blockIdx.x, sm, threadIdx.x, 0);
}

template <int G, int D>
cudaError_t launch_attn_t(AttnParams& p, cudaStream_t st, bool pdl) {
    dim3 grid(p.split ? p.max_chunks : 1, p.Hkv, p.B);
    return launch_k(attn_kernel<G, D>, grid, dim3(64), 0, st, pdl, p);
}

// ----------------------------------------------------------------------------
// Split-K attention, one 256-thread block per (page, kv head, request row).
// The 64-thread groups above leave one or two warps per SM to hide every
// shared-memory and shuffle latency of a page; here eight warps share it:
//   load    the page's keys (16-byte chunks rotated by row) and values with
//           asynchronous copies, eight per thread, and the G query rows;
//   scores  thread (position, dim quarter) forms G partial dot products, the
//           quarters are summed in shared memory;
//   softmax warp g takes query head g over the page's positions: page max m,
//           weights exp(s - m), their sum l;
//   values  thread (dim pair, head) accumulates the weighted value rows in
//           position order (with fewer than 512 outputs, groups of threads take
//           consecutive position ranges and their sums are added in order).
// The page's unnormalised state (o, m, l) goes to scratch; the last block of
// the (row, kv head) to arrive (completion ticket) combines every page's state
// with the usual softmax merge: weights exp(m_c - max m) / sum, outputs summed in
// page order, sixteen pages' loads in flight per thread (the first sixteen issued
// together with the loads of the page maxima and sums).
template <int G, int D>
struct AttnPageSmem {
    alignas(16) uint16_t sK[64 * D];
    alignas(16) uint16_t sV[64 * D];
    alignas(16) float sq[G][D];
    float sc[4][G][64];  // partial scores per dim quarter
    float sp[G][64];     // exp(s - m) of the page's positions
    // value partial sums of the position groups, when G x d < 512 (else unused)
    alignas(8) float pv[G * D < 512 ? 512 : 2];
    int last;
};

template <int G, int D>
__global__ void __launch_bounds__(256) attn_page_kernel(AttnParams p) {
    constexpr int NT = 256, CH = D / 8, P = 64;
    constexpr int PAIRS = D / 2, GS = NT / PAIRS, NG = (G + GS - 1) / GS;
    constexpr int PV_SPLIT = G * PAIRS >= NT ? 1 : NT / (G * PAIRS);
    static_assert(G * kMaxChunks * sizeof(float) <= sizeof(uint16_t) * 64 * D, "combine weights fit a stage");
    __shared__ AttnPageSmem<G, D> sm;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int chunk = blockIdx.x, kvh = blockIdx.y, row = blockIdx.z;
    pdl_trigger();
    // Lengths, positions, the page table and every cached key and value but the
    // newest position's were written before this step's first (non-overlapped)
    // launch: their loads go out before the wait for the kernel that wrote the
    // newest position's key and value (and the queries).
    const int ctx = p.ctx_lens ? p.ctx_lens[row] : p.positions[row] + 1;
    const int npages = (ctx + P - 1) / P;
    if (chunk >= npages) {
        pdl_wait();
        return;
    }
    const int req = p.row_req ? p.row_req[row] : row;
    const int nvalid = min(P, ctx - chunk * P);
    const int newest = ctx - 1 - chunk * P;  // row of the newest position in this page (< 0 or >= P: none)
    {
        const char* page = p.kv.base + p.kv.page_offsets[(int64_t)req * p.kv.max_pages + chunk] +
                           (uint64_t)p.kv.layer * p.kv.layer_page_bytes;
        const uint16_t* Kh = reinterpret_cast<const uint16_t*>(page) + (size_t)kvh * P * D;
        const uint16_t* Vh = reinterpret_cast<const uint16_t*>(page) + ((size_t)p.Hkv + kvh) * P * D;
        for (int i = tid; i < nvalid * CH; i += NT) {
            const int t = i / CH, c = i - t * CH;
            if (t == newest) continue;
            cp_async16(&sm.sK[(t * CH + ((c + t) & (CH - 1))) * 8], Kh + (size_t)t * D + c * 8);
            cp_async16(&sm.sV[(t * CH + c) * 8], Vh + (size_t)t * D + c * 8);
        }
        pdl_wait();
        if (newest >= 0 && newest < P)
            for (int c = tid; c < CH; c += NT) {
                cp_async16(&sm.sK[(newest * CH + ((c + newest) & (CH - 1))) * 8], Kh + (size_t)newest * D + c * 8);
                cp_async16(&sm.sV[(newest * CH + c) * 8], Vh + (size_t)newest * D + c * 8);
            }
        const float* qs = p.q + (size_t)row * p.Hq * D + (size_t)kvh * G * D;
        for (int i = tid; i < G * D / 4; i += NT)
            reinterpret_cast<float4*>(&sm.sq[0][0])[i] = ld_act4<false>(qs + 4 * i);
        cp_async_wait_all();
        __syncthreads();
    }
    {  // scores: a warp holds 32 consecutive positions of one dim quarter
        const int pos = tid & 63, dq = tid >> 6;
        float sc[G];
#pragma unroll
        for (int g = 0; g < G; ++g) sc[g] = 0.f;
        if (pos < nvalid) {
#pragma unroll
            for (int u = 0; u < CH / 4; ++u) {
                const int c = dq * (CH / 4) + u;
                const uint4 kk = *reinterpret_cast<const uint4*>(&sm.sK[(pos * CH + ((c + pos) & (CH - 1))) * 8]);
                const float kf[8] = {bf_lo(kk.x), bf_hi(kk.x), bf_lo(kk.y), bf_hi(kk.y),
                                     bf_lo(kk.z), bf_hi(kk.z), bf_lo(kk.w), bf_hi(kk.w)};
#pragma unroll
                for (int g = 0; g < G; ++g) {
                    const float4 qa = *reinterpret_cast<const float4*>(&sm.sq[g][c * 8]);
                    const float4 qb = *reinterpret_cast<const float4*>(&sm.sq[g][c * 8 + 4]);
                    float a = sc[g];
                    a = fmaf(qa.x, kf[0], a);
                    a = fmaf(qa.y, kf[1], a);
                    a = fmaf(qa.z, kf[2], a);
                    a = fmaf(qa.w, kf[3], a);
                    a = fmaf(qb.x, kf[4], a);
                    a = fmaf(qb.y, kf[5], a);
                    a = fmaf(qb.z, kf[6], a);
                    a = fmaf(qb.w, kf[7], a);
                    sc[g] = a;
                }
            }
        }
#pragma unroll
        for (int g = 0; g < G; ++g) sm.sc[dq][g][pos] = sc[g];
    }
    __syncthreads();
    float m_pg = 0.f, l_pg = 0.f;  // this warp's head (warp < G)
    if (warp < G) {
        const int g = warp;
        float s[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int t = lane + 32 * h;
            s[h] = t < nvalid ? (((sm.sc[0][g][t] + sm.sc[1][g][t]) + sm.sc[2][g][t]) + sm.sc[3][g][t]) * p.scale
                              : -INFINITY;
        }
        m_pg = warp_max(fmaxf(s[0], s[1]));  // finite: the page holds at least one position
        float lsum = 0.f;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const float e = lane + 32 * h < nvalid ? expf(s[h] - m_pg) : 0.f;
            sm.sp[g][lane + 32 * h] = e;
            lsum += e;
        }
        l_pg = warp_sum(lsum);
    }
    __syncthreads();
    const size_t hstride = (size_t)p.max_chunks * (D + 2);
    float* base = p.scratch + ((size_t)row * p.Hq + (size_t)kvh * G) * hstride;
    const int dp = tid % PAIRS;
    if constexpr (PV_SPLIT == 1) {
        const int g0 = tid / PAIRS;
        float acc[NG][2];
#pragma unroll
        for (int k = 0; k < NG; ++k) acc[k][0] = acc[k][1] = 0.f;
        for (int t = 0; t < nvalid; ++t) {
            const uint32_t vv = *reinterpret_cast<const uint32_t*>(&sm.sV[t * D + 2 * dp]);
            const float v0 = bf_lo(vv), v1 = bf_hi(vv);
#pragma unroll
            for (int k = 0; k < NG; ++k) {
                const int g = g0 + k * GS;
                if (g < G) {
                    const float pr = sm.sp[g][t];
                    acc[k][0] = fmaf(pr, v0, acc[k][0]);
                    acc[k][1] = fmaf(pr, v1, acc[k][1]);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < NG; ++k) {
            const int g = g0 + k * GS;
            if (g < G)
                *reinterpret_cast<float2*>(base + g * hstride + (size_t)chunk * (D + 2) + 2 * dp) =
                    make_float2(acc[k][0], acc[k][1]);
        }
    } else {
        // fewer outputs than threads (G x d / 2 < 256): PV_SPLIT thread groups take
        // consecutive position ranges, and group 0 adds the partial sums in order
        constexpr int SPAN = P / PV_SPLIT;
        const int rest = tid / PAIRS, g = rest % G, part = rest / G;
        const int t0 = part * SPAN, t1 = min(nvalid, t0 + SPAN);
        float a0 = 0.f, a1 = 0.f;
        for (int t = t0; t < t1; ++t) {
            const uint32_t vv = *reinterpret_cast<const uint32_t*>(&sm.sV[t * D + 2 * dp]);
            const float pr = sm.sp[g][t];
            a0 = fmaf(pr, bf_lo(vv), a0);
            a1 = fmaf(pr, bf_hi(vv), a1);
        }
        *reinterpret_cast<float2*>(&sm.pv[(part * G + g) * D + 2 * dp]) = make_float2(a0, a1);
        __syncthreads();
        if (part == 0) {
            float s0 = 0.f, s1 = 0.f;
#pragma unroll
            for (int q = 0; q < PV_SPLIT; ++q) {
                const float2 v = *reinterpret_cast<const float2*>(&sm.pv[(q * G + g) * D + 2 * dp]);
                s0 += v.x;
                s1 += v.y;
            }
            *reinterpret_cast<float2*>(base + g * hstride + (size_t)chunk * (D + 2) + 2 * dp) = make_float2(s0, s1);
        }
    }
    if (warp < G && lane == 0) {
        float* part = base + warp * hstride + (size_t)chunk * (D + 2);
        part[D] = m_pg;
        part[D + 1] = l_pg;
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) {
        int* cnt = p.counters + (size_t)row * p.Hq + kvh;
        const int ticket = atomicAdd(cnt, 1);
        sm.last = ticket == npages - 1;
        if (sm.last) atomicExch(cnt, 0);  // every page has arrived: reset for the next launch
    }
    __syncthreads();
    if (!sm.last) return;
    __threadfence();
    constexpr int NOUT = (G * D + NT - 1) / NT, PB = 16;
    // the first PB pages' partial outputs do not depend on the weights: their
    // loads go out together with those of the page maxima and sums
    float v[PB][NOUT];
#pragma unroll
    for (int u = 0; u < PB; ++u)
#pragma unroll
        for (int k = 0; k < NOUT; ++k) {
            const int e = tid + NT * k, g = e / D, j = e - g * D;
            v[u][k] = (e < G * D && u < npages) ? __ldcg(base + g * hstride + (size_t)u * (D + 2) + j) : 0.f;
        }
    // the stages are dead: page weights and denominators reuse them
    float(*s_w)[kMaxChunks] = reinterpret_cast<float(*)[kMaxChunks]>(&sm.sK[0]);
    float(*s_l)[kMaxChunks] = reinterpret_cast<float(*)[kMaxChunks]>(&sm.sV[0]);
    for (int i = tid; i < G * npages; i += NT) {
        const int g = i / npages, c = i - g * npages;
        const float* pc = base + g * hstride + (size_t)c * (D + 2);
        s_w[g][c] = __ldcg(pc + D);
        s_l[g][c] = __ldcg(pc + D + 1);
    }
    __syncthreads();
    if (warp < G) {
        const int g = warp;
        float mx = -INFINITY;
        for (int c = lane; c < npages; c += 32) mx = fmaxf(mx, s_w[g][c]);
        mx = warp_max(mx);
        float lsum = 0.f;
        for (int c = lane; c < npages; c += 32) {
            const float w = expf(s_w[g][c] - mx);
            s_w[g][c] = w;
            lsum = fmaf(s_l[g][c], w, lsum);
        }
        lsum = warp_sum(lsum);
        const float inv = 1.0f / lsum;
        for (int c = lane; c < npages; c += 32) s_w[g][c] *= inv;
    }
    __syncthreads();
    float o[NOUT];
#pragma unroll
    for (int k = 0; k < NOUT; ++k) o[k] = 0.f;
    for (int c0 = 0; c0 < npages; c0 += PB) {
        if (c0 > 0)
#pragma unroll
            for (int u = 0; u < PB; ++u)
#pragma unroll
                for (int k = 0; k < NOUT; ++k) {
                    const int e = tid + NT * k, g = e / D, j = e - g * D;
                    v[u][k] = (e < G * D && c0 + u < npages)
                                  ? __ldcg(base + g * hstride + (size_t)(c0 + u) * (D + 2) + j)
                                  : 0.f;
                }
#pragma unroll
        for (int u = 0; u < PB; ++u)
#pragma unroll
            for (int k = 0; k < NOUT; ++k) {
                const int e = tid + NT * k;
                if (e < G * D && c0 + u < npages) o[k] = fmaf(v[u][k], s_w[e / D][c0 + u], o[k]);
            }
    }
#pragma unroll
    for (int k = 0; k < NOUT; ++k) {
        const int e = tid + NT * k;
        if (e < G * D) {
            const size_t idx = (size_t)row * p.Hq * D + (size_t)kvh * G * D + e;
            store_o<D>(p, idx, o[k]);
        }
    }
}

template <int G, int D>
cudaError_t launch_attn_page_t(AttnParams& p, cudaStream_t st, bool pdl) {
    return launch_k(attn_page_kernel<G, D>, dim3(p.max_chunks, p.Hkv, p.B), dim3(256), 0, st, pdl, p);
}

template <int G, int D>
cudaError_t launch_attn_any(AttnParams& p, cudaStream_t st, bool pdl) {
    return p.split == kAttnWide ? launch_attn_page_t<G, D>(p, st, pdl) : launch_attn_t<G, D>(p, st, pdl);
}

// ----------------------------------------------------------------------------
// Persistent layer run (batch 1)
// ----------------------------------------------------------------------------
// The per-operation kernels of a batch-1 decode layer stream 34-235 MB each;
// every kernel boundary costs a ramp-up and a tail in which HBM idles, and
// attention leaves it idle altogether.  One cooperative launch keeps 2 blocks
// per SM resident through a run of resident layers: each phase hands out its
// tiles round-robin, grid barriers separate dependent phases, and before each
// barrier a block prefetches into L2 the first weight tile it will own in the
// next phase (weights never depend on activations), so the next phase starts on
// L2 hits.  During attention, the warps that hold no attention work prefetch
// the O-projection tiles.  Activations are read through L2 (ld.global.cg).
struct RunParams {
    const char* base[kMaxRunLayers];
    int n_layers, layer0;
    uint64_t off_g_attn, off_wqkv, off_wo, off_g_mlp, off_wg, off_wu, off_wd;
    int H, Hq, Hkv, d, F;
    float eps;
    float *x, *q, *o, *a;
    const int32_t* positions;
    KvView kv;
    float* scratch;
    int* counters;
    int max_chunks;
    unsigned* sync;  // [0] barrier counter, [1] error word, [2 ..] tile counters (4 per layer)
    uint32_t smem_bytes;
    int skip_block;             // fault injection: this block skips its first barrier arrival (-1: none)
    uint64_t barrier_limit_ns;  // bound of every barrier wait
    RopeFreqs rope;
};

__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Grid-wide barrier: every block arrives once per barrier on a monotonic
// counter.  The wait is bounded (limit_ns, 1 s by default); a block that gives
// up sets the error word, and a block that sees the error word stops waiting,
// so every block leaves the kernel instead of hanging.  Returns false on error.
// skip_block (fault injection for tests): that block does not arrive at the
// first barrier, so the barrier cannot complete and every wait runs out.
__device__ __forceinline__ bool grid_sync(unsigned* sync, unsigned& nsync, int* s_flag, int skip_block,
                                          uint64_t limit_ns) {
    __syncthreads();
    ++nsync;
    if (threadIdx.x == 0) {
        __threadfence();
        if (!(nsync == 1 && (int)blockIdx.x == skip_block)) atomicAdd(&sync[0], 1u);
        const unsigned target = nsync * gridDim.x;
        const uint64_t t0 = globaltimer_ns();
        int bad = 0;
        while (ld_acquire_u32(&sync[0]) < target) {
            if (*(volatile unsigned*)&sync[1]) {
                bad = 1;
                break;
            }
            if (globaltimer_ns() - t0 > limit_ns) {
                atomicCAS(&sync[1], 0u, 1u);
                bad = 1;
                break;
            }
        }
        __threadfence();
        *s_flag = bad;
    }
    __syncthreads();
    return *s_flag == 0;
}

template <int EPI>
__device__ __forceinline__ int tile_count(const GemvParams& p) {
    return (EPI == EPI_QKV || EPI == EPI_SWIGLU) ? (p.n_units + kTileRows / 2 - 1) / (kTileRows / 2)
                                                 : (p.N + kTileRows - 1) / kTileRows;
}

// Stages the phase's input row in shared memory (times the RMSNorm gain when
// the phase has one) and returns 1/rms (1 without a gain).  The sum of squares
// is accumulated in the per-tile path's order (each warp over its K slice, then
// lanes, then warps in order), so both paths produce the same bits.
__device__ __forceinline__ float stage_input(const GemvParams& p, float* sx, TileShared& sm) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int K = p.K;
    const int nj = (K + 255) >> 8, njw = (nj + kTileWarps - 1) / kTileWarps;
    const int j_begin = warp * njw, j_end = min(nj, j_begin + njw);
    const bool norm = p.g != nullptr;
    float ss = 0.f;
    for (int j = j_begin; j < j_end; ++j) {
        const int k = j * 256 + lane * 8;
        if (k >= K) continue;
        const float4 xa = ld_act4<true>(p.in + k);
        const float4 xb = ld_act4<true>(p.in + k + 4);
        float xv[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
        if (norm) {
            const uint4 gv = *reinterpret_cast<const uint4*>(p.g + k);
            const float gf[8] = {bf_lo(gv.x), bf_hi(gv.x), bf_lo(gv.y), bf_hi(gv.y),
                                 bf_lo(gv.z), bf_hi(gv.z), bf_lo(gv.w), bf_hi(gv.w)};
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                ss = fmaf(xv[e], xv[e], ss);
                xv[e] *= gf[e];
            }
        }
        *reinterpret_cast<float4*>(sx + k) = make_float4(xv[0], xv[1], xv[2], xv[3]);
        *reinterpret_cast<float4*>(sx + k + 4) = make_float4(xv[4], xv[5], xv[6], xv[7]);
    }
    if (norm) {
        const float v = warp_sum(ss);
        if (lane == 0) sm.ss[warp] = v;
    }
    __syncthreads();
    if (tid == 0) {
        float t = 0.f;
        if (norm)
            for (int w = 0; w < kTileWarps; ++w) t += sm.ss[w];
        sm.inv = norm ? 1.0f / sqrtf(t / (float)K + p.eps) : 1.0f;
    }
    __syncthreads();
    return sm.inv;
}

// This block's tiles of one phase.  The first tile is blockIdx.x; later ones
// are handed out by the phase's counter (first come, first served, so blocks
// that stream faster take more tiles), each fetched one tile ahead so that the
// next tile's first loads are issued while the current one reduces.  The input
// row is staged in shared memory when it fits (sx != nullptr).
template <int EPI>
__device__ __forceinline__ void run_tiles(const GemvParams& p, TileShared& tsm, float* sx, unsigned* ctr,
                                          int* s_next) {
    const int ntiles = tile_count<EPI>(p);
    int t = blockIdx.x;
    if (t >= ntiles) return;
    uint4 wa[kTileRows];
    tile_first_load<EPI>(p, t, wa);
    if (threadIdx.x == 0) *s_next = (int)(gridDim.x + atomicAdd(ctr, 1u));
    const float inv = sx ? stage_input(p, sx, tsm) : 1.f;
    __syncthreads();
    int nxt = *s_next;
    while (t < ntiles) {
        unsigned grabbed = 0;
        const bool more = nxt < ntiles;
        if (threadIdx.x == 0 && more) grabbed = gridDim.x + atomicAdd(ctr, 1u);
        if (sx)
            tile_gemv<EPI, true, true>(p, t, more ? nxt : -1, wa, tsm, sx, inv);
        else
            tile_gemv<EPI, true, false>(p, t, more ? nxt : -1, wa, tsm);
        if (threadIdx.x == 0) *s_next = more ? (int)grabbed : ntiles;
        __syncthreads();
        t = nxt;
        nxt = *s_next;
        __syncthreads();  // every thread has read s_next before it is rewritten
    }
}

enum { PH_QKV = 0, PH_O = 1, PH_GU = 2, PH_D = 3 };

template <int G, int D>
__global__ void __launch_bounds__(kTileWarps * 32, 2) decode_run_kernel(RunParams rp) {
    extern __shared__ __align__(16) unsigned char run_smem[];
    // attention: one AttnSmem per group; GEMV phases: the staged input row
    AttnSmem<G, D>* asm2 = reinterpret_cast<AttnSmem<G, D>*>(run_smem);
    float* sx_buf = reinterpret_cast<float*>(run_smem);
    __shared__ GemvParams s_gp[4];
    __shared__ AttnParams s_ap;
    __shared__ TileShared tsm;
    __shared__ int s_flag, s_next;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int qd = rp.Hq * rp.d, nqkv = (rp.Hq + 2 * rp.Hkv) * rp.d;
    // weight pointers of phase `ph` for layer `li` of the run
    auto set_layer = [&](int ph, int li) {
        const char* w = rp.base[li];
        GemvParams& g = s_gp[ph];
        if (ph == PH_QKV) {
            g.g = reinterpret_cast<const uint16_t*>(w + rp.off_g_attn);
            g.w0 = reinterpret_cast<const uint16_t*>(w + rp.off_wqkv);
            g.kv.layer = rp.layer0 + li;
        } else if (ph == PH_O) {
            g.w0 = reinterpret_cast<const uint16_t*>(w + rp.off_wo);
        } else if (ph == PH_GU) {
            g.g = reinterpret_cast<const uint16_t*>(w + rp.off_g_mlp);
            g.w0 = reinterpret_cast<const uint16_t*>(w + rp.off_wg);
            g.w1 = reinterpret_cast<const uint16_t*>(w + rp.off_wu);
        } else {
            g.w0 = reinterpret_cast<const uint16_t*>(w + rp.off_wd);
        }
    };
    if (tid == 0) {
        for (int ph = 0; ph < 4; ++ph) {
            GemvParams g{};
            g.B = 1;
            g.eps = rp.eps;
            s_gp[ph] = g;
        }
        GemvParams& q = s_gp[PH_QKV];
        q.in = rp.x;
        q.K = rp.H;
        q.N = nqkv;
        q.n_units = nqkv / 2;
        q.out = rp.q;
        q.Hq = rp.Hq;
        q.Hkv = rp.Hkv;
        q.d = rp.d;
        q.positions = rp.positions;
        q.kv = rp.kv;
        q.rope = rp.rope;
        GemvParams& o = s_gp[PH_O];
        o.in = rp.o;
        o.K = qd;
        o.N = rp.H;
        o.n_units = rp.H;
        o.out = rp.x;
        GemvParams& gu = s_gp[PH_GU];
        gu.in = rp.x;
        gu.K = rp.H;
        gu.N = rp.F;
        gu.n_units = rp.F;
        gu.out = rp.a;
        GemvParams& dn = s_gp[PH_D];
        dn.in = rp.a;
        dn.K = rp.F;
        dn.N = rp.H;
        dn.n_units = rp.H;
        dn.out = rp.x;
        for (int ph = 0; ph < 4; ++ph) set_layer(ph, 0);
        AttnParams a{};
        a.q = rp.q;
        a.kv = rp.kv;
        a.positions = rp.positions;
        a.B = 1;
        a.Hq = rp.Hq;
        a.Hkv = rp.Hkv;
        a.max_chunks = rp.max_chunks;
        a.scale = 1.0f / sqrtf((float)D);
        a.scratch = rp.scratch;
        a.counters = rp.counters;
        a.o = rp.o;
        a.split = kAttnSplit;
        s_ap = a;
    }
    __syncthreads();
    if (warp == 0) prefetch_tile<EPI_QKV>(s_gp[PH_QKV], blockIdx.x, lane);
    const int ctx = rp.positions[0] + 1;
    const int npages = (ctx + rp.kv.page_tokens - 1) / rp.kv.page_tokens;
    const int items = rp.Hkv * npages;
    unsigned nsync = 0;
    // the staged input row of a phase must fit the dynamic shared memory
    auto sx_for = [&](int K) { return (size_t)K * 4 <= rp.smem_bytes ? sx_buf : nullptr; };
    unsigned* ctr = rp.sync + 2;  // tile counters, 4 per layer, zeroed by the launcher
    for (int li = 0; li < rp.n_layers; ++li) {
        // ---- RMSNorm + QKV + RoPE + KV append
        run_tiles<EPI_QKV>(s_gp[PH_QKV], tsm, sx_for(rp.H), ctr + 4 * li + PH_QKV, &s_next);
        if (tid == 0) {
            s_ap.kv.layer = rp.layer0 + li;
            if (li + 1 < rp.n_layers) set_layer(PH_QKV, li + 1);
        }
        if (!grid_sync(rp.sync, nsync, &s_flag, rp.skip_block, rp.barrier_limit_ns)) return;
        // ---- split attention (groups = warp pairs 0-1 and 2-3); warps 4-7
        //      prefetch this block's O-projection tiles meanwhile
        if (warp < 4) {
            const int grp = warp >> 1;
            for (int i = blockIdx.x + grp * gridDim.x; i < items; i += 2 * gridDim.x)
                attn_group<G, D, true>(s_ap, 0, i / npages, i % npages, asm2[grp], tid & 63, 1 + grp);
        } else {
            // HBM is otherwise idle here: pull the O-projection tiles, then the
            // first gate/up tiles, into L2 (tiles blockIdx + k * grid; at most
            // 40 MB of each over the grid).  Whichever block later takes a tile
            // finds it in L2.
            const int k0 = warp - 4;
            const GemvParams& o = s_gp[PH_O];
            const GemvParams& gu = s_gp[PH_GU];
            const int nto = tile_count<EPI_RESID>(o), ntg = tile_count<EPI_SWIGLU>(gu);
            const uint64_t cap = 40ull << 20;
            const uint64_t ko = cap / ((uint64_t)kTileRows * o.K * 2 * gridDim.x);
            const uint64_t kg = cap / ((uint64_t)kTileRows * gu.K * 2 * gridDim.x);
            for (int kk = k0; kk < (int)(ko < 1 ? 1 : ko) && blockIdx.x + kk * gridDim.x < nto; kk += 4)
                prefetch_tile<EPI_RESID>(o, blockIdx.x + kk * gridDim.x, lane);
            for (int kk = k0; kk < (int)kg && blockIdx.x + kk * gridDim.x < ntg; kk += 4)
                prefetch_tile<EPI_SWIGLU>(gu, blockIdx.x + kk * gridDim.x, lane);
        }
        if (!grid_sync(rp.sync, nsync, &s_flag, rp.skip_block, rp.barrier_limit_ns)) return;
        // ---- O-projection + residual
        run_tiles<EPI_RESID>(s_gp[PH_O], tsm, sx_for(qd), ctr + 4 * li + PH_O, &s_next);
        if (warp == 0) prefetch_tile<EPI_SWIGLU>(s_gp[PH_GU], blockIdx.x, lane);
        if (tid == 0 && li + 1 < rp.n_layers) set_layer(PH_O, li + 1);
        if (!grid_sync(rp.sync, nsync, &s_flag, rp.skip_block, rp.barrier_limit_ns)) return;
        // ---- RMSNorm + gate/up SwiGLU
        run_tiles<EPI_SWIGLU>(s_gp[PH_GU], tsm, sx_for(rp.H), ctr + 4 * li + PH_GU, &s_next);
        if (warp == 0) prefetch_tile<EPI_RESID>(s_gp[PH_D], blockIdx.x, lane);
        if (tid == 0 && li + 1 < rp.n_layers) set_layer(PH_GU, li + 1);
        if (!grid_sync(rp.sync, nsync, &s_flag, rp.skip_block, rp.barrier_limit_ns)) return;
        // ---- down + residual
        run_tiles<EPI_RESID>(s_gp[PH_D], tsm, sx_for(rp.F), ctr + 4 * li + PH_D, &s_next);
        if (tid == 0 && li + 1 < rp.n_layers) set_layer(PH_D, li + 1);
        __syncthreads();
        if (warp == 0 && li + 1 < rp.n_layers) prefetch_tile<EPI_QKV>(s_gp[PH_QKV], blockIdx.x, lane);
        if (li + 1 < rp.n_layers && !grid_sync(rp.sync, nsync, &s_flag, rp.skip_block, rp.barrier_limit_ns)) return;
    }
}

// Dynamic shared memory of the layer-run kernel: the two attention groups'
// buffers, or the largest staged input row up to 96 KB (two blocks per SM).
template <int G, int D>
size_t run_smem_bytes(int H, int qd, int F) {
    size_t need = 2 * sizeof(AttnSmem<G, D>);
    const int kmax = H > qd ? (H > F ? H : F) : (qd > F ? qd : F);
    const size_t row = (size_t)kmax * 4;
    if (row <= (96u << 10) && row > need) need = row;
    return need;
}

template <int G, int D>
cudaError_t launch_run_t(RunParams& rp, cudaStream_t st) {
    const size_t smem = run_smem_bytes<G, D>(rp.H, rp.Hq * rp.d, rp.F);
    rp.smem_bytes = (uint32_t)smem;
    static size_t attr_smem = 0;
    static int grid = 0;
    if (attr_smem != smem) {  // per dynamic shared memory size: set the limit, size the grid from occupancy
        cudaError_t e = cudaFuncSetAttribute(decode_run_kernel<G, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        int dev = 0, sms = 0, per_sm = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_run_kernel<G, D>, kTileWarps * 32, smem);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) return cudaErrorInvalidConfiguration;
        grid = sms * (per_sm < 2 ? per_sm : 2);
        attr_smem = smem;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kTileWarps * 32);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeCooperative;  // all blocks co-resident: the grid barriers cannot deadlock
    at[0].val.cooperative = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, decode_run_kernel<G, D>, rp);
}

// ----------------------------------------------------------------------------
// QK-norm (Qwen3-style layers)
// ----------------------------------------------------------------------------
struct QkNormParams {
    const float* raw;  // [rows][(Hq + 2 Hkv) d] unrotated projections
    int rows, Hq, Hkv, d, with_v;
    const uint16_t *g_q, *g_k;  // [d] gains
    float eps;
    const int32_t* positions;
    const int32_t* row_req;
    float* q_out;  // [rows][Hq d]
    KvView kv;
    RopeFreqs rope;
};

// One block of d/2 threads per (row, head): RMSNorm of the head's d values
// (gain g_q for query heads, g_k for key heads), the rotation at the row's
// position, then the QKV epilogue's stores: queries to q_out (fp32), keys to
// the KV cache (bf16); with_v: value heads are copied to the cache unchanged.
__global__ void __launch_bounds__(64) qk_norm_rope_kernel(QkNormParams p) {
    __shared__ float s_ss[2];
    pdl_trigger();
    pdl_wait();
    const int h = blockIdx.x, b = blockIdx.y;
    const int half = p.d >> 1, i = threadIdx.x;
    const float* raw = p.raw + (size_t)b * (p.Hq + 2 * p.Hkv) * p.d + (size_t)h * p.d;
    float v0 = raw[i], v1 = raw[i + half];
    const int pos = p.positions[b];
    if (h < p.Hq + p.Hkv) {
        float ss = warp_sum(fmaf(v0, v0, v1 * v1));
        if ((i & 31) == 0) s_ss[i >> 5] = ss;
        __syncthreads();
        ss = s_ss[0] + (half > 32 ? s_ss[1] : 0.f);
        const float inv = 1.0f / sqrtf(ss / (float)p.d + p.eps);
        const uint16_t* g = h < p.Hq ? p.g_q : p.g_k;
        v0 = v0 * inv * bf2f(g[i]);
        v1 = v1 * inv * bf2f(g[i + half]);
        float cf, sf;
        rope_cos_sin(pos, p.rope.inv_freq[i], &cf, &sf);
        const float r0 = v0 * cf - v1 * sf, r1 = v1 * cf + v0 * sf;
        v0 = r0;
        v1 = r1;
    }
    if (h < p.Hq) {
        float* q = p.q_out + (size_t)b * p.Hq * p.d + (size_t)h * p.d;
        q[i] = v0;
        q[i + half] = v1;
    } else {
        const int req = p.row_req ? p.row_req[b] : b;
        const bool is_v = h >= p.Hq + p.Hkv;
        const int kh = h - p.Hq - (is_v ? p.Hkv : 0);
        uint16_t* row = reinterpret_cast<uint16_t*>(kv_row(p.kv, req, pos, is_v ? 1 : 0, kh, p.Hkv, p.d));
        row[i] = f2bf(v0);
        row[i + half] = f2bf(v1);
    }
}

// ----------------------------------------------------------------------------
// Embedding gather and generator
// ----------------------------------------------------------------------------
__global__ void embed_kernel(const uint16_t* E, const int32_t* tokens, int H, int V, float* x) {
    pdl_trigger();
    pdl_wait();
    const int b = blockIdx.x;
    const int tok = tokens[b];
    const bool ok = tok >= 0 && tok < V;
    const uint4* row = reinterpret_cast<const uint4*>(E + (size_t)(ok ? tok : 0) * H);
    float4* out = reinterpret_cast<float4*>(x + (size_t)b * H);
    for (int i = threadIdx.x; i < H / 8; i += blockDim.x) {  // 8 bf16 per 16-byte load
        const uint4 v = ok ? row[i] : make_uint4(0, 0, 0, 0);
        out[2 * i] = make_float4(bf_lo(v.x), bf_hi(v.x), bf_lo(v.y), bf_hi(v.y));
        out[2 * i + 1] = make_float4(bf_lo(v.z), bf_hi(v.z), bf_lo(v.w), bf_hi(v.w));
    }
}

// SplitMix64 (Steele, Lea & Flood 2014) used as a counter-based generator:
// output k of the stream seeded with s is mix(s + (k+1) * golden gamma).
__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t k) {
    uint64_t z = seed + (k + 1ull) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// Irwin-Hall (n = 4) sum of the four 16-bit fields, centred, scaled so the
// standard deviation is 0.02 (weights) or 1 + 0.02 z (gains); bf16 RNE.
__device__ __forceinline__ uint16_t gen_elem(uint64_t seed, uint32_t tensor_id, uint64_t index, int kind) {
    uint64_t r = splitmix64_at(seed, ((uint64_t)tensor_id << 40) | index);
    int s = (int)(r & 0xffffu) + (int)((r >> 16) & 0xffffu) + (int)((r >> 32) & 0xffffu) + (int)(r >> 48);
    float z = __fmul_rn(__int2float_rn(s - 131070), 0x1p-16f);
    float w = __fmul_rn(z, 0x1.1bc77ap-5f);
    if (kind == 1) w = __fadd_rn(1.0f, w);
    return f2bf(w);
}

__global__ void advance_kernel(int32_t* pos, int B) {
    pdl_trigger();
    pdl_wait();
    if ((int)threadIdx.x < B) pos[threadIdx.x] += 1;
}

__global__ void generate_kernel(uint16_t* out, uint64_t n, uint64_t first, uint64_t seed, uint32_t tensor_id,
                                int kind) {
    uint64_t i = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x;
    const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
    for (; i < n; i += stride) out[i] = gen_elem(seed, tensor_id, first + i, kind);
}

// 128-bit streaming reads of n16 vectors, four in flight per thread; one
// xor-fold per block keeps every load live.
__global__ void __launch_bounds__(256) read_stream_kernel(const uint4* src, uint64_t n16, uint32_t* sink) {
    __shared__ uint32_t s_x[8];
    uint32_t x = 0;
    const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
    uint64_t i = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x;
    for (; i + 3 * stride < n16; i += 4 * stride) {
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = ld_stream(reinterpret_cast<const uint16_t*>(src + i + u * stride));
#pragma unroll
        for (int u = 0; u < 4; ++u) x ^= v[u].x ^ v[u].y ^ v[u].z ^ v[u].w;
    }
    for (; i < n16; i += stride) {
        const uint4 v = ld_stream(reinterpret_cast<const uint16_t*>(src + i));
        x ^= v.x ^ v.y ^ v.z ^ v.w;
    }
    for (int o = 16; o; o >>= 1) x ^= __shfl_xor_sync(0xffffffffu, x, o);
    if ((threadIdx.x & 31) == 0) s_x[threadIdx.x >> 5] = x;
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t t = 0;
        for (int w = 0; w < 8; ++w) t ^= s_x[w];
        sink[blockIdx.x] = t;
    }
}

}  // namespace

// ----------------------------------------------------------------------------
// launchers
// ----------------------------------------------------------------------------
cudaError_t launch_qkv_rope(const float* x, const uint16_t* g, const uint16_t* wqkv, int B, int H, int Hq, int Hkv,
                            int d, float eps, float theta, const int32_t* positions, float* q_out, KvView kv,
                            const int32_t* row_req, cudaStream_t st, bool pdl, bool w_host, float* qk_raw) {
    GemvParams p{};
    p.w_host = w_host;
    p.qk_raw = qk_raw;
    p.in = x;
    p.g = g;
    p.w0 = wqkv;
    p.B = B;
    p.K = H;
    p.N = (Hq + 2 * Hkv) * d;
    p.n_units = p.N / 2;
    p.eps = eps;
    p.out = q_out;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.d = d;
    p.rope = rope_freqs(theta, d);
    p.positions = positions;
    p.row_req = row_req;
    p.kv = kv;
    return launch_gemv<EPI_QKV>(p, st, pdl);
}

cudaError_t launch_resid_gemv(const float* in, const uint16_t* w, int B, int N, int K, float* x, cudaStream_t st,
                              bool pdl, bool w_host, bool prefetch_waves) {
    GemvParams p{};
    p.w_host = w_host;
    if (prefetch_waves && !w_host) {  // two block-tile blocks are resident per SM
        static int sms = 0;
        if (!sms) {
            int dev = 0;
            if (cudaGetDevice(&dev) != cudaSuccess ||
                cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
                sms = 0;
        }
        p.pf_stride = 2 * sms;
    }
    p.in = in;
    p.w0 = w;
    p.B = B;
    p.K = K;
    p.N = N;
    p.n_units = N;
    p.out = x;
    return launch_gemv<EPI_RESID>(p, st, pdl);
}

cudaError_t launch_gate_up(const float* x, const uint16_t* g, const uint16_t* wg, const uint16_t* wu, int B, int H,
                           int F, float eps, float* a, cudaStream_t st, bool pdl, bool w_host) {
    GemvParams p{};
    p.w_host = w_host;
    p.in = x;
    p.g = g;
    p.w0 = wg;
    p.w1 = wu;
    p.B = B;
    p.K = H;
    p.N = F;
    p.n_units = F;
    p.eps = eps;
    p.out = a;
    return launch_gemv<EPI_SWIGLU>(p, st, pdl);
}

RopeFreqs rope_freqs(float theta, int d) {
    RopeFreqs f{};
    for (int i = 0; i < d / 2 && i < 64; ++i) f.inv_freq[i] = pow((double)theta, -2.0 * (double)i / (double)d);
    return f;
}

size_t lm_head_scratch_bytes(int B, int V) {
    (void)B;
    // one key per (block, batch slot) for at most ceil(V/2/kWarps) blocks and 8 slots
    size_t blocks = ((size_t)V / 2 + kWarps) / kWarps + 1;
    return blocks * 8 * sizeof(uint64_t);
}

cudaError_t launch_lm_head(const float* x, const uint16_t* g, const uint16_t* w, int B, int H, int V, float eps,
                           float* z, float* logits, int32_t* tokens, void* scratch, cudaStream_t st, bool pdl) {
    GemvParams p{};
    p.in = x;
    p.g = g;
    p.w0 = w;
    p.B = B;
    p.K = H;
    p.N = V;
    p.n_units = (V + 1) / 2;
    p.eps = eps;
    p.out = logits;
    p.z = z;
    p.keys = reinterpret_cast<uint64_t*>(scratch);
    int nblocks = 0;
    cudaError_t e = launch_gemv<EPI_LOGITS>(p, st, pdl, &nblocks);
    if (e != cudaSuccess) return e;
    int BT = B <= 1 ? 1 : B <= 2 ? 2 : B <= 4 ? 4 : 8;
    return launch_k(argmax_reduce_kernel, dim3(B), dim3(256), 0, st, true, (const uint64_t*)p.keys, nblocks, BT, B,
                    tokens);
}

static size_t attention_partial_floats(int B, int Hq, int d, int max_ctx, int page_tokens) {
    size_t chunks = ((size_t)max_ctx + page_tokens - 1) / page_tokens;
    return ((size_t)B * Hq * chunks * (d + 2) + 63) / 64 * 64;
}

size_t attention_scratch_floats(int B, int Hq, int d, int max_ctx, int page_tokens) {
    return attention_partial_floats(B, Hq, d, max_ctx, page_tokens) + (size_t)B * Hq;  // + int counters
}

int* attention_counters(float* scratch, int B, int Hq, int d, int max_ctx, int page_tokens) {
    return reinterpret_cast<int*>(scratch + attention_partial_floats(B, Hq, d, max_ctx, page_tokens));
}

cudaError_t launch_attention(const float* q, KvView kv, const int32_t* ctx_lens, const int32_t* positions,
                             const int32_t* row_req, int B, int Hq, int Hkv, int d, int max_ctx, bool split,
                             float* scratch, void* o, bool o_split, cudaStream_t st, bool pdl, int scratch_rows,
                             bool wide) {
    AttnParams p{};
    p.q = q;
    p.kv = kv;
    p.ctx_lens = ctx_lens;
    p.positions = positions;
    p.row_req = row_req;
    p.B = B;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.max_chunks = (max_ctx + kv.page_tokens - 1) / kv.page_tokens;
    if (split && p.max_chunks > kMaxChunks) return cudaErrorInvalidValue;
    p.scale = 1.0f / sqrtf((float)d);
    p.scratch = scratch;
    if (scratch_rows < B) scratch_rows = B;
    p.counters = split ? attention_counters(scratch, scratch_rows, Hq, d, max_ctx, kv.page_tokens) : nullptr;
    p.o = o;
    p.o_split = o_split ? 1 : 0;
    p.split = split ? kAttnSplit : kAttnSingle;
    if (split && wide) p.split = kAttnWide;
    const int G = Hq / Hkv;
    if (d == 128) {
        switch (G) {
            case 1: return launch_attn_any<1, 128>(p, st, pdl);
            case 2: return launch_attn_any<2, 128>(p, st, pdl);
            case 4: return launch_attn_any<4, 128>(p, st, pdl);
            case 8: return launch_attn_any<8, 128>(p, st, pdl);
        }
    } else if (d == 64) {
        switch (G) {
            case 1: return launch_attn_any<1, 64>(p, st, pdl);
            case 2: return launch_attn_any<2, 64>(p, st, pdl);
            case 4: return launch_attn_any<4, 64>(p, st, pdl);
            case 8: return launch_attn_any<8, 64>(p, st, pdl);
        }
    }
    return cudaErrorInvalidValue;
}

cudaError_t launch_qk_norm_rope(const float* raw, int rows, int Hq, int Hkv, int d, bool with_v, const uint16_t* g_q,
                                const uint16_t* g_k, float eps, float theta, const int32_t* positions,
                                const int32_t* row_req, float* q_out, KvView kv, cudaStream_t st, bool pdl) {
    if (rows < 1 || (d != 64 && d != 128)) return cudaErrorInvalidValue;
    QkNormParams p{};
    p.raw = raw;
    p.rows = rows;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.d = d;
    p.with_v = with_v ? 1 : 0;
    p.g_q = g_q;
    p.g_k = g_k;
    p.eps = eps;
    p.positions = positions;
    p.row_req = row_req;
    p.q_out = q_out;
    p.kv = kv;
    p.rope = rope_freqs(theta, d);
    return launch_k(qk_norm_rope_kernel, dim3(Hq + Hkv + (with_v ? Hkv : 0), rows), dim3(d / 2), 0, st, pdl, p);
}

bool decode_run_supported(int Hq, int Hkv, int d) {
    const int G = Hkv > 0 ? Hq / Hkv : 0;
    return (d == 64 || d == 128) && (G == 1 || G == 2 || G == 4 || G == 8) && Hq == G * Hkv;
}

cudaError_t launch_decode_run(const DecodeRunArgs& a, cudaStream_t st) {
    if (a.n_layers < 1 || a.n_layers > kMaxRunLayers || !decode_run_supported(a.Hq, a.Hkv, a.d) || !a.sync)
        return cudaErrorInvalidValue;
    RunParams rp{};
    for (int i = 0; i < a.n_layers; ++i) rp.base[i] = a.base[i];
    rp.n_layers = a.n_layers;
    rp.layer0 = a.layer0;
    rp.off_g_attn = a.off_g_attn;
    rp.off_wqkv = a.off_wqkv;
    rp.off_wo = a.off_wo;
    rp.off_g_mlp = a.off_g_mlp;
    rp.off_wg = a.off_wg;
    rp.off_wu = a.off_wu;
    rp.off_wd = a.off_wd;
    rp.H = a.H;
    rp.Hq = a.Hq;
    rp.Hkv = a.Hkv;
    rp.d = a.d;
    rp.F = a.F;
    rp.eps = a.eps;
    rp.x = a.x;
    rp.q = a.q;
    rp.o = a.o;
    rp.a = a.a;
    rp.positions = a.positions;
    rp.kv = a.kv;
    rp.scratch = a.attn_scratch;
    rp.max_chunks = (a.max_ctx + a.kv.page_tokens - 1) / a.kv.page_tokens;
    if (rp.max_chunks > kMaxChunks) return cudaErrorInvalidValue;
    rp.counters = attention_counters(a.attn_scratch, a.scratch_rows < 1 ? 1 : a.scratch_rows, a.Hq, a.d, a.max_ctx,
                                     a.kv.page_tokens);
    rp.sync = a.sync;
    rp.skip_block = a.skip_block;
    rp.barrier_limit_ns = a.barrier_limit_us ? (uint64_t)a.barrier_limit_us * 1000ull : 1000000000ull;
    rp.rope = rope_freqs(a.theta, a.d);
    // the barrier counter and the tile counters; the error word (sync[1]) is kept
    cudaError_t e = cudaMemsetAsync(a.sync, 0, sizeof(unsigned), st);
    if (e == cudaSuccess) e = cudaMemsetAsync(a.sync + 2, 0, sizeof(unsigned) * 4 * a.n_layers, st);
    if (e != cudaSuccess) return e;
    const int G = a.Hq / a.Hkv;
    if (a.d == 128) {
        switch (G) {
            case 1: return launch_run_t<1, 128>(rp, st);
            case 2: return launch_run_t<2, 128>(rp, st);
            case 4: return launch_run_t<4, 128>(rp, st);
            case 8: return launch_run_t<8, 128>(rp, st);
        }
    } else {
        switch (G) {
            case 1: return launch_run_t<1, 64>(rp, st);
            case 2: return launch_run_t<2, 64>(rp, st);
            case 4: return launch_run_t<4, 64>(rp, st);
            case 8: return launch_run_t<8, 64>(rp, st);
        }
    }
    return cudaErrorInvalidValue;
}

cudaError_t launch_embed(const uint16_t* embed, const int32_t* tokens, int B, int H, int V, float* x,
                         cudaStream_t st, bool pdl) {
    return launch_k(embed_kernel, dim3(B), dim3(256), 0, st, pdl, embed, tokens, H, V, x);
}

cudaError_t launch_read_stream(const void* src, uint64_t bytes, int blocks, uint32_t* sink, cudaStream_t st) {
    return launch_k(read_stream_kernel, dim3(blocks), dim3(256), 0, st, false, reinterpret_cast<const uint4*>(src),
                    bytes / 16, sink);
}

cudaError_t launch_advance(int32_t* positions, int B, cudaStream_t st, bool pdl) {
    return launch_k(advance_kernel, dim3(1), dim3(32), 0, st, pdl, positions, B);
}

cudaError_t launch_generate(uint16_t* out, uint64_t n, uint64_t first, uint64_t seed, uint32_t tensor_id, int kind,
                            cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    uint64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 32) blocks = 152 * 32;
    return launch_k(generate_kernel, dim3((unsigned)blocks), dim3(256), 0, st, false, out, n, first, seed, tensor_id,
                    kind);
}

}  // namespace loip
