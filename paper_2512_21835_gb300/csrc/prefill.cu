// prefill.cu -- prefill of M prompt tokens per layer: bf16 GEMMs with fp32
// accumulation and fused epilogues (query/key rotation + KV-cache write,
// residual add, SwiGLU), and the row-wise RMSNorm that feeds them.
//
// Activations entering a projection are rounded to bf16 (the GEMM operand
// type); accumulation, rotation, softmax and the residual stream stay fp32.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "internal.h"

namespace loip {
namespace {

__device__ __forceinline__ float bf2f(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }
__device__ __forceinline__ uint16_t f2bf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }

__global__ void rmsnorm_bf16_kernel(const float* x, const uint16_t* g, int H, float eps, uint16_t* y) {
    __shared__ float red[32];
    const int m = blockIdx.x;
    const float* xr = x + (size_t)m * H;
    float ss = 0.f;
    for (int k = threadIdx.x; k < H; k += blockDim.x) ss = fmaf(xr[k], xr[k], ss);
    for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    if (threadIdx.x < 32) {
        float t = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
        for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (threadIdx.x == 0) red[0] = 1.0f / sqrtf(t / (float)H + eps);
    }
    __syncthreads();
    const float inv = red[0];
    for (int k = threadIdx.x; k < H; k += blockDim.x) y[(size_t)m * H + k] = f2bf(xr[k] * inv * bf2f(g[k]));
}

__global__ void gather_rows_kernel(const float* x, const int32_t* rows, int H, float* out) {
    const int i = blockIdx.x;
    const float* src = x + (size_t)rows[i] * H;
    for (int k = threadIdx.x; k < H; k += blockDim.x) out[(size_t)i * H + k] = src[k];
}

// ---------------------------------------------------------------------------
// Tiled GEMM  C[M, N] = A[M, K] * W[N, K]^T  (both K-contiguous bf16)
// ---------------------------------------------------------------------------
constexpr int BM = 128, BN = 128, BK = 32;
enum { G_QKV = 0, G_RESID = 1, G_SWIGLU = 2 };

struct GemmParams {
    const uint16_t* A;
    const uint16_t* W0;
    const uint16_t* W1;  // SwiGLU: up rows fill tile columns 64..127
    int M, N, K;
    float* x;       // RESID
    uint16_t* a;    // SWIGLU output [M, F]
    float* q;       // QKV
    int Hq, Hkv, d;
    float theta;
    const int32_t* positions;
    const int32_t* row_req;
    KvView kv;
};

template <int EPI>
__device__ __forceinline__ const uint16_t* w_row(const GemmParams& p, int tile_n0, int r, bool& ok) {
    if (EPI == G_SWIGLU) {
        int f = tile_n0 / 2 + (r & 63);
        ok = f < p.N;
        return (r < 64 ? p.W0 : p.W1) + (size_t)f * p.K;
    }
    int n = tile_n0 + r;
    ok = n < p.N;
    return p.W0 + (size_t)n * p.K;
}

template <int EPI>
__global__ void __launch_bounds__(256) gemm_kernel(GemmParams p) {
    extern __shared__ __align__(16) float smem[];
    float* As = smem;            // [BK][BM]
    float* Ws = smem + BK * BM;  // [BK][BN]
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;

    for (int k0 = 0; k0 < p.K; k0 += BK) {
        // 128 rows x 32 k = 512 16-byte vectors per operand; 2 per thread
#pragma unroll
        for (int it = 0; it < 2; ++it) {
            int v = tid + it * 256;
            int r = v >> 2, kv = (v & 3) * 8;
            int k = k0 + kv;
            uint4 va = make_uint4(0, 0, 0, 0), vw = make_uint4(0, 0, 0, 0);
            if (m0 + r < p.M && k < p.K) va = *reinterpret_cast<const uint4*>(p.A + (size_t)(m0 + r) * p.K + k);
            bool ok;
            const uint16_t* wr = w_row<EPI>(p, n0, r, ok);
            if (ok && k < p.K) vw = *reinterpret_cast<const uint4*>(wr + k);
            const uint32_t wa[4] = {va.x, va.y, va.z, va.w}, ww[4] = {vw.x, vw.y, vw.z, vw.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                As[(kv + 2 * e) * BM + r] = __uint_as_float(wa[e] << 16);
                As[(kv + 2 * e + 1) * BM + r] = __uint_as_float(wa[e] & 0xffff0000u);
                Ws[(kv + 2 * e) * BN + r] = __uint_as_float(ww[e] << 16);
                Ws[(kv + 2 * e + 1) * BN + r] = __uint_as_float(ww[e] & 0xffff0000u);
            }
        }
        __syncthreads();
#pragma unroll 4
        for (int kk = 0; kk < BK; ++kk) {
            float4 a0 = *reinterpret_cast<const float4*>(&As[kk * BM + ty * 4]);
            float4 a1 = *reinterpret_cast<const float4*>(&As[kk * BM + 64 + ty * 4]);
            float4 b0 = *reinterpret_cast<const float4*>(&Ws[kk * BN + tx * 4]);
            float4 b1 = *reinterpret_cast<const float4*>(&Ws[kk * BN + 64 + tx * 4]);
            const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
        __syncthreads();
    }

    // stage the tile in shared memory so epilogues can pair columns
    float* Cs = smem;  // [BM][BN + 1]
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            int r = (i < 4 ? ty * 4 + i : 64 + ty * 4 + i - 4);
            int c = (j < 4 ? tx * 4 + j : 64 + tx * 4 + j - 4);
            Cs[r * (BN + 1) + c] = acc[i][j];
        }
    __syncthreads();

    if (EPI == G_RESID) {
        for (int e = tid; e < BM * BN; e += 256) {
            int r = e / BN, c = e % BN;
            int m = m0 + r, n = n0 + c;
            if (m < p.M && n < p.N) p.x[(size_t)m * p.N + n] += Cs[r * (BN + 1) + c];
        }
    } else if (EPI == G_SWIGLU) {
        const int F = p.N, f0 = n0 / 2;
        for (int e = tid; e < BM * 64; e += 256) {
            int r = e / 64, c = e % 64;
            int m = m0 + r, f = f0 + c;
            if (m < p.M && f < F) {
                float gt = Cs[r * (BN + 1) + c], ut = Cs[r * (BN + 1) + 64 + c];
                float silu = gt / (1.0f + expf(-gt));
                p.a[(size_t)m * F + f] = f2bf(silu * ut);
            }
        }
    } else {  // G_QKV: the tile spans whole heads (d divides BN)
        const int half = p.d >> 1;
        for (int e = tid; e < BM * (BN / 2); e += 256) {
            int r = e / (BN / 2), pi = e % (BN / 2);
            int hb = (pi / half) * p.d, i = pi % half;
            int m = m0 + r, n = n0 + hb;
            if (m >= p.M || n >= p.N) continue;
            int h = n / p.d;
            float v0 = Cs[r * (BN + 1) + hb + i], v1 = Cs[r * (BN + 1) + hb + i + half];
            const int pos = p.positions[m];
            if (h < p.Hq + p.Hkv) {
                double freq = pow((double)p.theta, -2.0 * (double)i / (double)p.d);
                double s, c;
                sincos((double)pos * freq, &s, &c);
                float cf = (float)c, sf = (float)s;
                float r0 = v0 * cf - v1 * sf, r1 = v1 * cf + v0 * sf;
                v0 = r0;
                v1 = r1;
            }
            if (h < p.Hq) {
                float* q = p.q + (size_t)m * p.Hq * p.d + (size_t)h * p.d;
                q[i] = v0;
                q[i + half] = v1;
            } else {
                const int req = p.row_req[m];
                const bool is_v = h >= p.Hq + p.Hkv;
                const int kh = h - p.Hq - (is_v ? p.Hkv : 0);
                int page = pos / p.kv.page_tokens, t = pos - page * p.kv.page_tokens;
                char* base = p.kv.base + p.kv.page_offsets[(int64_t)req * p.kv.max_pages + page] +
                             (uint64_t)p.kv.layer * p.kv.layer_page_bytes;
                uint16_t* row = reinterpret_cast<uint16_t*>(
                    base + ((uint64_t)((is_v ? p.Hkv : 0) + kh) * p.kv.page_tokens + t) * (uint64_t)p.d * 2u);
                row[i] = f2bf(v0);
                row[i + half] = f2bf(v1);
            }
        }
    }
}

constexpr size_t kGemmSmem = (size_t)BM * (BN + 1) * sizeof(float);

template <int EPI>
cudaError_t launch_gemm(GemmParams& p, int n_cols, cudaStream_t st) {
    static bool attr = false;
    if (!attr) {
        cudaFuncSetAttribute(gemm_kernel<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemmSmem);
        attr = true;
    }
    dim3 grid((n_cols + BN - 1) / BN, (p.M + BM - 1) / BM);
    gemm_kernel<EPI><<<grid, 256, kGemmSmem, st>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rmsnorm_bf16(const float* x, const uint16_t* g, int M, int H, float eps, uint16_t* y,
                                cudaStream_t st) {
    if (M <= 0) return cudaSuccess;
    rmsnorm_bf16_kernel<<<M, 256, 0, st>>>(x, g, H, eps, y);
    return cudaGetLastError();
}

cudaError_t launch_gather_rows(const float* x, const int32_t* rows, int n, int H, float* out, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    gather_rows_kernel<<<n, 256, 0, st>>>(x, rows, H, out);
    return cudaGetLastError();
}

cudaError_t launch_gemm_qkv_rope(const uint16_t* y, const uint16_t* wqkv, int M, int H, int Hq, int Hkv, int d,
                                 float theta, const int32_t* positions, const int32_t* row_req, float* q, KvView kv,
                                 cudaStream_t st) {
    if (BN % d != 0) return cudaErrorInvalidValue;
    GemmParams p{};
    p.A = y;
    p.W0 = wqkv;
    p.M = M;
    p.N = (Hq + 2 * Hkv) * d;
    p.K = H;
    p.q = q;
    p.Hq = Hq;
    p.Hkv = Hkv;
    p.d = d;
    p.theta = theta;
    p.positions = positions;
    p.row_req = row_req;
    p.kv = kv;
    return launch_gemm<G_QKV>(p, p.N, st);
}

cudaError_t launch_gemm_resid(const uint16_t* a, const uint16_t* w, int M, int N, int K, float* x, cudaStream_t st) {
    GemmParams p{};
    p.A = a;
    p.W0 = w;
    p.M = M;
    p.N = N;
    p.K = K;
    p.x = x;
    return launch_gemm<G_RESID>(p, N, st);
}

cudaError_t launch_gemm_swiglu(const uint16_t* y, const uint16_t* wg, const uint16_t* wu, int M, int H, int F,
                               uint16_t* a, cudaStream_t st) {
    GemmParams p{};
    p.A = y;
    p.W0 = wg;
    p.W1 = wu;
    p.M = M;
    p.N = F;
    p.K = H;
    p.a = a;
    // each 128-column tile covers 64 gate rows and the matching 64 up rows
    return launch_gemm<G_SWIGLU>(p, 2 * ((F + 63) / 64) * 64, st);
}

}  // namespace loip
