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
// same order, the same two shuffle trees), with the row held in registers: its
// loads are all in flight at once and the row is read once.  H <= 256 * kRowRegs.
constexpr int kRowRegs = 32;
__global__ void __launch_bounds__(256) rmsnorm_split_reg_kernel(const float* x, const uint16_t* g, int H, float eps,
                                                                uint16_t* y) {
    __shared__ float red[32];
    const int m = blockIdx.x;
    const float* xr = x + (size_t)m * H;
    float v[kRowRegs];
#pragma unroll
    for (int j = 0; j < kRowRegs; ++j) {
        const int k = threadIdx.x + 256 * j;
        v[j] = k < H ? xr[k] : 0.f;
    }
    float ss = 0.f;
#pragma unroll
    for (int j = 0; j < kRowRegs; ++j)
        if (threadIdx.x + 256 * j < H) ss = fmaf(v[j], v[j], ss);
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
#pragma unroll
    for (int j = 0; j < kRowRegs; ++j) {
        const int k = threadIdx.x + 256 * j;
        if (k >= H) break;
        const float f = v[j] * inv * bf2f(g[k]);
        const uint16_t hi = f2bf(f);
        y[(size_t)m * H + k] = hi;
        y[plane + (size_t)m * H + k] = f2bf(f - bf2f(hi));
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
    if (H <= 256 * kRowRegs)
        rmsnorm_split_reg_kernel<<<M, 256, 0, st>>>(x, g, H, eps, y);
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
