// prefill.cu -- the row-wise pieces of a prefill pass: the RMSNorm that feeds
// each tensor-core projection and a row gather.  The projections themselves
// are in gemm_tc.cu.  The normed rows are computed in fp32 and written as the
// GEMM's split operand, a pair of bf16 planes: hi = bf16(y) and lo =
// bf16(y - hi), so the projection sees y to ~2^-17 relative (the residual
// stream stays fp32).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "internal.h"

namespace loip {
namespace {

__device__ __forceinline__ float bf2f(uint16_t h) { return __uint_as_float((uint32_t)h << 16); }
__device__ __forceinline__ uint16_t f2bf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }

__global__ void rmsnorm_split_kernel(const float* x, const uint16_t* g, int H, float eps, uint16_t* y) {
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
    const size_t plane = (size_t)gridDim.x * H;  // rows = gridDim.x
    for (int k = threadIdx.x; k < H; k += blockDim.x) {
        const float v = xr[k] * inv * bf2f(g[k]);
        const uint16_t hi = f2bf(v);
        y[(size_t)m * H + k] = hi;
        y[plane + (size_t)m * H + k] = f2bf(v - bf2f(hi));
    }
}

// The same arithmetic, bit for bit (each thread sums the same elements in the
// same order, the same two shuffle trees), with 16-byte loads of the row into
// registers and shared memory (the sum reads it back in the original order) and
// 8-byte stores of four bf16 per plane.  H % 4 == 0, H <= 4 * 256 * kRowVec.
constexpr int kRowVec = 8;
__global__ void __launch_bounds__(256) rmsnorm_split_vec_kernel(const float* x, const uint16_t* g, int H, float eps,
                                                                uint16_t* y) {
    __shared__ float red[32];
    __shared__ float4 row4[256 * kRowVec];
    const int m = blockIdx.x, H4 = H >> 2;
    const float4* xr = reinterpret_cast<const float4*>(x + (size_t)m * H);
    float4 v[kRowVec];
#pragma unroll
    for (int j = 0; j < kRowVec; ++j) {
        const int k = threadIdx.x + 256 * j;
        v[j] = k < H4 ? xr[k] : make_float4(0.f, 0.f, 0.f, 0.f);
        if (k < H4) row4[k] = v[j];
    }
    __syncthreads();
    const float* row = reinterpret_cast<const float*>(row4);
    float ss = 0.f;
    for (int k = threadIdx.x; k < H; k += 256) ss = fmaf(row[k], row[k], ss);
    for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    if (threadIdx.x < 32) {
        float t = threadIdx.x < 8 ? red[threadIdx.x] : 0.f;
        for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (threadIdx.x == 0) red[0] = 1.0f / sqrtf(t / (float)H + eps);
    }
    __syncthreads();
    const float inv = red[0];
    const size_t plane = (size_t)gridDim.x * H;  // rows = gridDim.x
    uint2* hi_row = reinterpret_cast<uint2*>(y + (size_t)m * H);
    uint2* lo_row = reinterpret_cast<uint2*>(y + plane + (size_t)m * H);
    const uint2* g4 = reinterpret_cast<const uint2*>(g);
#pragma unroll
    for (int j = 0; j < kRowVec; ++j) {
        const int k = threadIdx.x + 256 * j;
        if (k >= H4) break;
        const uint2 gg = g4[k];
        const float f[4] = {v[j].x * inv * bf2f((uint16_t)(gg.x & 0xffffu)), v[j].y * inv * bf2f((uint16_t)(gg.x >> 16)),
                            v[j].z * inv * bf2f((uint16_t)(gg.y & 0xffffu)), v[j].w * inv * bf2f((uint16_t)(gg.y >> 16))};
        uint32_t hi[4], lo[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            hi[i] = f2bf(f[i]);
            lo[i] = f2bf(f[i] - bf2f((uint16_t)hi[i]));
        }
        hi_row[k] = make_uint2(hi[0] | hi[1] << 16, hi[2] | hi[3] << 16);
        lo_row[k] = make_uint2(lo[0] | lo[1] << 16, lo[2] | lo[3] << 16);
    }
}

__global__ void gather_rows_kernel(const float* x, const int32_t* rows, int H, float* out) {
    const int i = blockIdx.x;
    const float* src = x + (size_t)rows[i] * H;
    for (int k = threadIdx.x; k < H; k += blockDim.x) out[(size_t)i * H + k] = src[k];
}

}  // namespace

cudaError_t launch_rmsnorm_split(const float* x, const uint16_t* g, int M, int H, float eps, uint16_t* y,
                                 cudaStream_t st) {
    if (M <= 0) return cudaSuccess;
    if (H % 4 == 0 && H <= 4 * 256 * kRowVec && !((uintptr_t)x & 15) && !((uintptr_t)g & 7) && !((uintptr_t)y & 7))
        rmsnorm_split_vec_kernel<<<M, 256, 0, st>>>(x, g, H, eps, y);
    else
        rmsnorm_split_kernel<<<M, 256, 0, st>>>(x, g, H, eps, y);
    return cudaGetLastError();
}

cudaError_t launch_gather_rows(const float* x, const int32_t* rows, int n, int H, float* out, cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    gather_rows_kernel<<<n, 256, 0, st>>>(x, rows, H, out);
    return cudaGetLastError();
}

}  // namespace loip
