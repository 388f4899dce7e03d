// Fully connected layer (Sec. IV-A; split over output neurons in Sec. IV-B):
// y[b][o] = sum_i x[b][i] * W[o][i] + bias[o], int32 output, no compression.
// One warp per input row b: lanes stride over K four bytes at a time with
// dp4a.u32.s32 (u8 activations x s8 weights), then a warp reduction per output.
// Outputs are processed 16 at a time so any m works.
#include <algorithm>
#include <cstdint>
#include <mutex>

#include "internal.h"

namespace qnn {
namespace {

constexpr int kOutChunk = 16;

__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int c)
{
    int d;
    asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}

template <bool VEC>
__global__ void __launch_bounds__(256) linear_kernel(int n, int k, int m, const uint8_t *x, const int8_t *w,
                                                     const int32_t *bias, int32_t *y)
{
    const int row = blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= n) return;
    const uint8_t *xr = x + static_cast<long long>(row) * k;
    for (int o0 = 0; o0 < m; o0 += kOutChunk) {
        int acc[kOutChunk];
#pragma unroll
        for (int j = 0; j < kOutChunk; ++j) acc[j] = 0;
        if (VEC) {
            const uint32_t *xw = reinterpret_cast<const uint32_t *>(xr);
            for (int i4 = lane; i4 < k / 4; i4 += 32) {
                const uint32_t xv = __ldg(xw + i4);
#pragma unroll
                for (int j = 0; j < kOutChunk; ++j)
                    if (o0 + j < m)
                        acc[j] = dp4a_us(xv, __ldg(reinterpret_cast<const uint32_t *>(w + static_cast<long long>(o0 + j) * k) + i4), acc[j]);
            }
        } else {
            for (int i = lane; i < k; i += 32) {
                const int xv = xr[i];
#pragma unroll
                for (int j = 0; j < kOutChunk; ++j)
                    if (o0 + j < m) acc[j] += xv * w[static_cast<long long>(o0 + j) * k + i];
            }
        }
#pragma unroll
        for (int j = 0; j < kOutChunk; ++j) {
            int v = acc[j];
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
            if (lane == j && o0 + j < m) y[static_cast<long long>(row) * m + o0 + j] = v + (bias ? bias[o0 + j] : 0);
        }
    }
}

// Rows of 16-byte vectors, weights staged once per block in shared memory: each
// warp takes whole input rows (grid-stride), lanes stride over the row 16 bytes
// at a time, and every output takes four dp4a per vector from the shared copy
// of its weight row (consecutive lanes read consecutive vectors, no bank
// conflicts).  Outputs go kOutChunk at a time.
constexpr int kSmemRowsMax = 200 * 1024;  // weight bytes kept in shared memory

__global__ void __launch_bounds__(256) linear_smem_kernel(int n, int k, int m, const uint8_t *x, const int8_t *w,
                                                          const int32_t *bias, int32_t *y)
{
    extern __shared__ uint4 wsh[];  // [m][k/16]
    const int kv = k / 16;
    const uint4 *wg = reinterpret_cast<const uint4 *>(w);
    for (int i = threadIdx.x; i < m * kv; i += blockDim.x) wsh[i] = __ldg(wg + i);
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int warps = gridDim.x * (blockDim.x >> 5);
    for (int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); row < n; row += warps) {
        const uint4 *xr = reinterpret_cast<const uint4 *>(x + static_cast<long long>(row) * k);
        for (int o0 = 0; o0 < m; o0 += kOutChunk) {
            int acc[kOutChunk];
#pragma unroll
            for (int j = 0; j < kOutChunk; ++j) acc[j] = 0;
            for (int i = lane; i < kv; i += 32) {
                const uint4 xv = __ldg(xr + i);
#pragma unroll
                for (int j = 0; j < kOutChunk; ++j) {
                    if (o0 + j < m) {
                        const uint4 wv = wsh[(o0 + j) * kv + i];
                        int a = dp4a_us(xv.x, wv.x, acc[j]);
                        a = dp4a_us(xv.y, wv.y, a);
                        a = dp4a_us(xv.z, wv.z, a);
                        acc[j] = dp4a_us(xv.w, wv.w, a);
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < kOutChunk; ++j) {
                int v = acc[j];
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
                if (lane == j && o0 + j < m) y[static_cast<long long>(row) * m + o0 + j] = v + (bias ? bias[o0 + j] : 0);
            }
        }
    }
}

}  // namespace

cudaError_t launch_linear(int n, int k, int m, const uint8_t *x, const int8_t *w, const int32_t *bias, int32_t *y,
                          cudaStream_t st)
{
    if (n == 0) return cudaSuccess;
    const size_t wbytes = static_cast<size_t>(m) * k;
    if (k % 16 == 0 && (reinterpret_cast<uintptr_t>(x) % 16) == 0 && (reinterpret_cast<uintptr_t>(w) % 16) == 0 &&
        wbytes <= static_cast<size_t>(kSmemRowsMax)) {
        // opt-in shared memory above 48 KB, raised once per device
        static std::mutex mu;
        static bool raised[64] = {};
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return e;
        {
            std::lock_guard<std::mutex> lock(mu);
            if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
            if (!raised[dev]) {
                e = cudaFuncSetAttribute(linear_smem_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemRowsMax);
                if (e != cudaSuccess) return e;
                raised[dev] = true;
            }
        }
        // enough warps to cover the rows, at most a few blocks per SM
        const int blocks = static_cast<int>(std::min<long long>((n + 7) / 8, 4ll * device_sm_count()));
        linear_smem_kernel<<<blocks, 256, wbytes, st>>>(n, k, m, x, w, bias, y);
        return cudaGetLastError();
    }
    const unsigned grid = static_cast<unsigned>((n + 7) / 8);
    const bool vec = k % 4 == 0 && (reinterpret_cast<uintptr_t>(x) % 4) == 0 && (reinterpret_cast<uintptr_t>(w) % 4) == 0;
    if (vec) linear_kernel<true><<<grid, 256, 0, st>>>(n, k, m, x, w, bias, y);
    else linear_kernel<false><<<grid, 256, 0, st>>>(n, k, m, x, w, bias, y);
    return cudaGetLastError();
}

}  // namespace qnn
