// attn_tc.cu -- causal prefill attention on the 5th-generation tensor cores.
//
// The prefill's attention (every prompt token against the cached keys and
// values of its request up to its own position: grouped-query attention with a
// causal mask) is a dense contraction over 128-row query tiles, so it runs as
// tcgen05 MMAs: S = Q K^T into tensor memory, the softmax on the CUDA cores,
// O_blk = P V into tensor memory, one key page (64 positions) at a time.
//
// Tile.  One CTA per (query tile, kv head).  A query tile is up to P_T = 128 / G
// consecutive positions of one request (G = Hq / Hkv query heads share the kv
// head), so its 128 MMA rows are (position, query head) pairs, row = pi * G + gi:
// every row of the tile attends over the same key pages, read once per CTA.
//
// Precision.  The operands of kind::f16 are bf16; the queries (fp32) and the
// probabilities P (fp32) are each given as a split pair hi = bf16(v), lo =
// bf16(v - hi), two MMAs per K step, so the products carry ~16 significant
// bits; keys and values are the cache's bf16 values exactly.  The tensor core
// sums at most one page per MMA group (its truncating accumulation stays
// short); each page's O_blk is added to fp32 registers with the online-softmax
// rescale (round to nearest).  The output is written as the next projection's
// split operand.
//
// Shared memory (bf16, K-major, 128-byte swizzle: 16-byte chunk c of row r at
// r * 128 + ((c ^ (r & 7)) * 16), 8-row atoms of 1024 bytes):
//   Q_hi, Q_lo   [128 rows][D]        D/64 slabs of 16 KB each
//   K            [64 keys][D]         D/64 slabs of 8 KB, two buffers (the next
//                                     page loads while this one is used)
//   V^T          [D rows][64 keys]    slabs of D * 128 bytes, two buffers
//                                     (transposed by the threads, 8 x 8 blocks
//                                     in registers)
//   P_hi, P_lo   [128 rows][64 keys]  one slab of 16 KB each
// Tensor memory: S [128 x 64] fp32 at column 0, O_blk [128 x D] at column 128.
//
// Threads: 8 warps; warp w owns TMEM lanes 32 (w % 4) .. + 31 (one query row
// per lane) and half hh = w / 4 of the row's columns (S columns 32 hh .. +31,
// O columns hh D/2 .. +D/2-1).  Thread 0 issues the MMAs.  Every wait is
// bounded (2 s of %globaltimer); on timeout the CTA records an error code,
// waits for its MMAs, frees its tensor memory and returns.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "internal.h"

namespace loip {

__device__ int g_attn_tc_error;  // first failure code of any tensor-core attention launch (0 = none)

namespace {

constexpr int kAttnThreads = 256;
constexpr int kKeys = 64;            // keys per block (one KV page)
constexpr uint32_t kTmemCols = 256;  // S at 0..63, O_blk at 128..128+D-1
constexpr uint32_t kOCol = 128;

template <int D>
struct AttnTcSmem {
    static constexpr int SLABS = D / 64;
    static constexpr int Q_SLAB = 128 * 128;  // bytes: 128 rows x 64 bf16
    static constexpr int K_SLAB = 64 * 128;
    static constexpr int QHI = 0;
    static constexpr int QLO = QHI + SLABS * Q_SLAB;
    static constexpr int KB = QLO + SLABS * Q_SLAB;  // two K buffers: page kb and page kb + 1
    static constexpr int KBUF = SLABS * K_SLAB;
    static constexpr int VT = KB + 2 * KBUF;  // two V^T slabs: page kb and page kb + 1
    static constexpr int VTBUF = D * 128;
    static constexpr int PHI = VT + 2 * VTBUF;
    static constexpr int PLO = PHI + Q_SLAB;
    static constexpr int RED = PLO + Q_SLAB;  // float [2][128] row maxima of the two column halves
    static constexpr int BAR = RED + 2 * 128 * 4;
    static constexpr int BYTES = BAR + 64;
    static constexpr int ALLOC = BYTES + 1024;  // + alignment of the dynamic window
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ uint16_t f2bf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }
__device__ __forceinline__ float bf2f(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }
__device__ __forceinline__ uint32_t swz(int r, int c) { return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4)); }

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
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
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (global_ns() - t0 > 2000000000ull) return false;
    }
}
// kind::f16 instruction descriptor: fp32 accumulator, bf16 A and B, both
// K-major, M = 128, N = n
__host__ __device__ constexpr uint32_t idesc(int n) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
}
__device__ __forceinline__ void umma(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t id, uint32_t acc) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
            tmem_d),
        "l"(adesc), "l"(bdesc), "r"(id), "r"(acc)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr) {  // K-major, 128-byte rows, 128-byte swizzle
    uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
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
// 16-byte copy; with n = 0 nothing is read and the destination is zero-filled
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t n) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n) : "memory");
}

struct AttnTcParams {
    const float* q;      // [M, Hq * D] fp32
    KvView kv;
    const int4* tiles;   // {row0, n_rows, request, pos0}
    int Hq, Hkv, M;
    float scale;
    uint16_t* o;         // split pair [2][M][Hq * D]
};

template <int G, int D>
__global__ void __launch_bounds__(kAttnThreads, 1) attn_tc_kernel(const AttnTcParams p) {
    using S = AttnTcSmem<D>;
    constexpr int PT = 128 / G;  // positions per tile
    constexpr int DH = D / 2;    // O columns per thread
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    float* red = reinterpret_cast<float*>(sm + S::RED);
    uint64_t* bar = reinterpret_cast<uint64_t*>(sm + S::BAR);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + S::BAR + 24);
    // completion of: S = Q K^T; O_blk = P V; everything issued (error path)
    const uint32_t sbase = smem_u32(sm), mbar_s = smem_u32(bar), mbar_pv = smem_u32(bar + 1),
                   mbar_end = smem_u32(bar + 2);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int4 tile = p.tiles[blockIdx.x];
    const int g = blockIdx.y;  // kv head
    const int row0 = tile.x, nrows = tile.y, req = tile.z, pos0 = tile.w;
    const int qd = p.Hq * D;

    if (tid == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(mbar_s) : "memory");
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(mbar_pv) : "memory");
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(mbar_end) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    // ---- Q tile -> split pair, swizzled (thread: one row, one 32-element quarter of D/2)
    {
        const int r = tid >> 1, part = tid & 1;  // row, half of D
        const int pi = r / G, gi = r - pi * G;
        const bool live = pi < nrows;
        const float* qr = p.q + (size_t)(row0 + (live ? pi : 0)) * qd + (size_t)(g * G + gi) * D;
#pragma unroll
        for (int c8 = 0; c8 < DH / 8; ++c8) {  // 8 elements = one 16-byte chunk
            const int e0 = part * DH + c8 * 8;
            float v[8];
            if (live) {
                const float4 a = *reinterpret_cast<const float4*>(qr + e0);
                const float4 b = *reinterpret_cast<const float4*>(qr + e0 + 4);
                v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w; v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
            } else {
#pragma unroll
                for (int i = 0; i < 8; ++i) v[i] = 0.f;
            }
            uint32_t hi[4], lo[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint16_t h0 = f2bf(v[2 * i]), h1 = f2bf(v[2 * i + 1]);
                hi[i] = (uint32_t)h0 | ((uint32_t)h1 << 16);
                lo[i] = (uint32_t)f2bf(v[2 * i] - bf2f(h0)) | ((uint32_t)f2bf(v[2 * i + 1] - bf2f(h1)) << 16);
            }
            const int slab = e0 >> 6, c = (e0 & 63) >> 3;
            const uint32_t off = (uint32_t)(slab * S::Q_SLAB) + swz(r, c);
            *reinterpret_cast<uint4*>(sm + S::QHI + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
            *reinterpret_cast<uint4*>(sm + S::QLO + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_slot;

    const int q4 = warp & 3, hh = warp >> 2;
    const int r = q4 * 32 + lane;  // this thread's row
    const int pi = r / G;
    const bool live = pi < nrows;
    const int my_pos = pos0 + (live ? pi : 0);
    const uint32_t t_row = tmem + ((uint32_t)(q4 * 32) << 16);
    float o[DH];
#pragma unroll
    for (int j = 0; j < DH; ++j) o[j] = 0.f;
    float m_run = -INFINITY, l_run = 0.f;
    uint32_t phase_s = 0, phase_pv = 0;
    bool ok = true;
    const int last_pos = pos0 + nrows - 1;
    const int nkb = last_pos / kKeys + 1;
    const char* kv_layer = p.kv.base + (uint64_t)p.kv.layer * p.kv.layer_page_bytes;

    // Positions past the tile's last one hold no key yet (the page may keep
    // anything there): their K and V are zero-filled, so that their zero
    // weights in P meet finite values (0 x NaN would spoil the row).
    auto page_at = [&](int kb) { return kv_layer + p.kv.page_offsets[(int64_t)req * p.kv.max_pages + kb]; };
    // K page kb -> K buffer b, K-major slabs (cp.async)
    auto load_k = [&](int kb, int b) {
        const char* kp = page_at(kb) + (size_t)g * kKeys * D * 2;
        const int n_keys = last_pos - kb * kKeys + 1;  // valid keys in this page (>= 1)
        for (int i = tid; i < kKeys * (D / 8); i += kAttnThreads) {
            const int key = i / (D / 8), c = i - key * (D / 8);  // 16-byte chunk c of the key's row
            cp_async16(sbase + S::KB + (uint32_t)(b * S::KBUF + (c >> 3) * S::K_SLAB) + swz(key, c & 7),
                       kp + (size_t)key * D * 2 + c * 16, key < n_keys ? 16u : 0u);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    // V page kb -> registers.  The page is cut into 8 x 8 blocks (keys 8 kc ..,
    // dims 8 c ..); thread 2 blk + h holds dims 4h .. 4h+3 of block blk's 8 keys.
    constexpr int kVThreads = 2 * 8 * (D / 8);
    uint2 vin[8];
    auto load_v = [&](int kb) {
        if (tid >= kVThreads) return;
        const int blk = tid >> 1, h = tid & 1, kc = blk & 7, c = blk >> 3;
        const char* vp = page_at(kb) + (size_t)(p.Hkv + g) * kKeys * D * 2 + c * 16 + h * 8;
        const int n_keys = last_pos - kb * kKeys + 1;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int key = 8 * kc + i;
            vin[i] = key < n_keys ? *reinterpret_cast<const uint2*>(vp + (size_t)key * D * 2) : make_uint2(0u, 0u);
        }
    };
    // registers -> V^T slab: row dd = 8 c + j holds the 8 keys of block blk as
    // one 16-byte chunk (kc)
    auto store_vt = [&](int b) {
        if (tid >= kVThreads) return;
        const int blk = tid >> 1, h = tid & 1, kc = blk & 7, c = blk >> 3;
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) {
            const uint32_t sel = (jj & 1) ? 0x7632u : 0x5410u;  // high or low halves of the two words
            uint32_t w[4];
#pragma unroll
            for (int k2 = 0; k2 < 4; ++k2) {
                const uint32_t a = (jj >> 1) ? vin[2 * k2].y : vin[2 * k2].x;
                const uint32_t b = (jj >> 1) ? vin[2 * k2 + 1].y : vin[2 * k2 + 1].x;
                w[k2] = __byte_perm(a, b, sel);  // keys 2 k2, 2 k2 + 1 of dim 4h + jj
            }
            *reinterpret_cast<uint4*>(sm + S::VT + b * S::VTBUF + swz(8 * c + 4 * h + jj, kc)) =
                make_uint4(w[0], w[1], w[2], w[3]);
        }
    };
    // S = (Q_hi + Q_lo) K^T of page kb (K buffer kb & 1), completion on mbar_s
    auto issue_s = [&](int kb) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
        for (int k = 0; k < D / 16; ++k) {
            const uint32_t qo = (uint32_t)((k >> 2) * S::Q_SLAB);
            const uint32_t ko = (uint32_t)((kb & 1) * S::KBUF + (k >> 2) * S::K_SLAB);
            const uint64_t bd = sdesc(sbase + S::KB + ko) + 2 * (k & 3);
            umma(tmem, sdesc(sbase + S::QHI + qo) + 2 * (k & 3), bd, idesc(kKeys), k != 0);
            umma(tmem, sdesc(sbase + S::QLO + qo) + 2 * (k & 3), bd, idesc(kKeys), 1u);
        }
        umma_commit(mbar_s);
    };
    // Pipeline: while the CUDA cores run page kb's softmax and O update, the
    // tensor core runs S of page kb + 1 (issued right behind P V of page kb),
    // and the loads of page kb + 2 are in flight.
    load_k(0, 0);
    load_v(0);
    store_vt(0);
    asm volatile("cp.async.wait_all;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // generic-proxy writes -> the tensor core
    __syncthreads();
    if (tid == 0) issue_s(0);
    if (nkb > 1) {
        load_k(1, 1);
        load_v(1);
    }

    for (int kb = 0; kb < nkb && ok; ++kb) {
        const bool more = kb + 1 < nkb;
        if (tid == 0 && !mbar_wait(mbar_s, phase_s)) {
            atomicCAS(&g_attn_tc_error, 0, 1);
            ok = false;
        }
        phase_s ^= 1;
        ok = __syncthreads_and(ok);
        if (!ok) break;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        // ---- online softmax over this page (scores of my 32 keys)
        float s[32];
        {
            float a[16], b[16];
            tmem_ld16(t_row + (uint32_t)(hh * 32), a);
            tmem_ld16(t_row + (uint32_t)(hh * 32 + 16), b);
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                s[j] = a[j];
                s[16 + j] = b[j];
            }
        }
        float mx = -INFINITY;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const int key = kb * kKeys + hh * 32 + j;
            s[j] = (live && key <= my_pos) ? s[j] * p.scale : -INFINITY;
            mx = fmaxf(mx, s[j]);
        }
        red[hh * 128 + r] = mx;
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();
        const float m_new = fmaxf(m_run, fmaxf(red[r], red[128 + r]));
        // a live row has its key 0 in page 0, so m_new is finite from the first page on
        const float alpha = live ? expf(m_run - m_new) : 0.f;
        float lsum = 0.f;
        uint32_t phi[16], plo[16];
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
            const float p0 = live ? expf(s[j] - m_new) : 0.f, p1 = live ? expf(s[j + 1] - m_new) : 0.f;
            lsum += p0 + p1;
            const uint16_t h0 = f2bf(p0), h1 = f2bf(p1);
            phi[j / 2] = (uint32_t)h0 | ((uint32_t)h1 << 16);
            plo[j / 2] = (uint32_t)f2bf(p0 - bf2f(h0)) | ((uint32_t)f2bf(p1 - bf2f(h1)) << 16);
        }
        m_run = live ? m_new : m_run;
        l_run = l_run * alpha + lsum;
#pragma unroll
        for (int c = 0; c < 4; ++c) {  // my keys hh*32 .. +31 = chunks 4 hh .. 4 hh + 3 of the row
            const uint32_t off = swz(r, hh * 4 + c);
            *reinterpret_cast<uint4*>(sm + S::PHI + off) =
                make_uint4(phi[4 * c], phi[4 * c + 1], phi[4 * c + 2], phi[4 * c + 3]);
            *reinterpret_cast<uint4*>(sm + S::PLO + off) =
                make_uint4(plo[4 * c], plo[4 * c + 1], plo[4 * c + 2], plo[4 * c + 3]);
        }
        // ---- the next page's V^T (its slab was last read by P V of page kb - 1,
        // complete) and K (landed)
        if (more) {
            store_vt((kb + 1) & 1);
            asm volatile("cp.async.wait_all;" ::: "memory");
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();
        // ---- O_blk = (P_hi + P_lo) V, then S of the next page behind it
        if (tid == 0) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t vt = sbase + S::VT + (uint32_t)((kb & 1) * S::VTBUF);
#pragma unroll
            for (int k = 0; k < kKeys / 16; ++k) {
                const uint64_t bd = sdesc(vt) + 2 * k;
                umma(tmem + kOCol, sdesc(sbase + S::PHI) + 2 * k, bd, idesc(D), k != 0);
                umma(tmem + kOCol, sdesc(sbase + S::PLO) + 2 * k, bd, idesc(D), 1u);
            }
            umma_commit(mbar_pv);
            if (more) issue_s(kb + 1);
        }
        // ---- page kb + 2 into the K buffer S of page kb used (complete) and registers
        if (kb + 2 < nkb) {
            load_k(kb + 2, kb & 1);
            load_v(kb + 2);
        }
        if (tid == 0 && !mbar_wait(mbar_pv, phase_pv)) {
            atomicCAS(&g_attn_tc_error, 0, 2);
            ok = false;
        }
        phase_pv ^= 1;
        ok = __syncthreads_and(ok);
        if (!ok) break;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        // ---- O = O * alpha + O_blk (my D/2 columns), in fp32 registers.  The next
        // P V writes O_blk only after the barriers of the next page's softmax.
#pragma unroll
        for (int j0 = 0; j0 < DH; j0 += 16) {
            float v[16];
            tmem_ld16(t_row + kOCol + (uint32_t)(hh * DH + j0), v);
#pragma unroll
            for (int j = 0; j < 16; ++j) o[j0 + j] = fmaf(o[j0 + j], alpha, v[j]);
        }
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    }
    // a wait that gave up can leave the next page's copies in flight
    asm volatile("cp.async.wait_all;" ::: "memory");
    if (ok) {
        // l of the row = both halves' sums
        red[hh * 128 + r] = l_run;
        __syncthreads();
        const float inv = live ? 1.0f / (red[r] + red[128 + r]) : 0.f;
        if (live) {
            const size_t plane = (size_t)p.M * qd;
            uint16_t* orow = p.o + (size_t)(row0 + pi) * qd + (size_t)(g * G + (r - pi * G)) * D + hh * DH;
#pragma unroll
            for (int j = 0; j < DH; j += 8) {
                uint32_t hi[4], lo[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float v0 = o[j + 2 * i] * inv, v1 = o[j + 2 * i + 1] * inv;
                    const uint16_t h0 = f2bf(v0), h1 = f2bf(v1);
                    hi[i] = (uint32_t)h0 | ((uint32_t)h1 << 16);
                    lo[i] = (uint32_t)f2bf(v0 - bf2f(h0)) | ((uint32_t)f2bf(v1 - bf2f(h1)) << 16);
                }
                *reinterpret_cast<uint4*>(orow + j) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                *reinterpret_cast<uint4*>(orow + plane + j) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
        }
    } else if (tid == 0) {
        // a commit of everything issued so far, so no MMA is in flight when the
        // tensor memory is released (bounded like every other wait)
        umma_commit(mbar_end);
        mbar_wait(mbar_end, 0);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

template <int G, int D>
cudaError_t launch_t(const AttnTcParams& p, int n_tiles, cudaStream_t st) {
    constexpr int SMEM = AttnTcSmem<D>::ALLOC;
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<G, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    attn_tc_kernel<G, D><<<dim3(n_tiles, p.Hkv), kAttnThreads, SMEM, st>>>(p);
    return cudaGetLastError();
}

}  // namespace

int attention_tc_tile_positions(int Hq, int Hkv) { return Hkv > 0 ? 128 / (Hq / Hkv) : 0; }

cudaError_t launch_attention_tc(const float* q, KvView kv, const int4* tiles, int n_tiles, int M, int Hq, int Hkv,
                                int d, uint16_t* o, cudaStream_t st) {
    if (n_tiles <= 0) return cudaSuccess;
    if (kv.page_tokens != kKeys || Hkv < 1 || Hq % Hkv) return cudaErrorInvalidValue;
    AttnTcParams p{};
    p.q = q;
    p.kv = kv;
    p.tiles = tiles;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.M = M;
    p.scale = 1.0f / sqrtf((float)d);
    p.o = o;
    const int G = Hq / Hkv;
    if (d == 128) {
        switch (G) {
            case 1: return launch_t<1, 128>(p, n_tiles, st);
            case 2: return launch_t<2, 128>(p, n_tiles, st);
            case 4: return launch_t<4, 128>(p, n_tiles, st);
            case 8: return launch_t<8, 128>(p, n_tiles, st);
        }
    } else if (d == 64) {
        switch (G) {
            case 1: return launch_t<1, 64>(p, n_tiles, st);
            case 2: return launch_t<2, 64>(p, n_tiles, st);
            case 4: return launch_t<4, 64>(p, n_tiles, st);
            case 8: return launch_t<8, 64>(p, n_tiles, st);
        }
    }
    return cudaErrorInvalidValue;
}

cudaError_t attention_tc_error(int* code) { return cudaMemcpyFromSymbol(code, g_attn_tc_error, sizeof(int)); }

}  // namespace loip
