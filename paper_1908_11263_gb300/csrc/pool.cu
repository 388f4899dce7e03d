// Max-pooling on packed NHWC activations (Sec. IV-A; split over output pixels as
// in Sec. IV-B).  One thread produces 16 output bytes (pixels of whole 16-byte
// vectors: 128-bit loads and a field-wise vmax at any Q) or one output byte (any
// layout).  No padding, floor output size.
#include <cstdint>

#include "device.cuh"
#include "internal.h"

namespace qnn {
namespace {

// One thread produces one 16-byte vector of an output pixel (pixels whose bytes
// are whole 16-byte vectors).
template <int BITS>
__global__ void __launch_bounds__(256) maxpool_vec_kernel(int n, int h, int w, int vec_per_pix, int k, int s, int oh,
                                                          int ow, const uint4 *x, uint4 *y)
{
    const long long total = static_cast<long long>(n) * oh * ow * vec_per_pix;
    const long long gid = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (gid >= total) return;
    const int v = static_cast<int>(gid % vec_per_pix);
    const long long pix = gid / vec_per_pix;
    const int ox = static_cast<int>(pix % ow);
    const int oy = static_cast<int>((pix / ow) % oh);
    const int b = static_cast<int>(pix / (static_cast<long long>(ow) * oh));
    uint4 best = make_uint4(0, 0, 0, 0);
    for (int i = 0; i < k; ++i)
        for (int j = 0; j < k; ++j) {
            const long long src = ((static_cast<long long>(b) * h + oy * s + i) * w + ox * s + j) * vec_per_pix + v;
            const uint4 t = __ldg(x + src);
            best.x = max_fields<BITS>(best.x, t.x);
            best.y = max_fields<BITS>(best.y, t.y);
            best.z = max_fields<BITS>(best.z, t.z);
            best.w = max_fields<BITS>(best.w, t.w);
        }
    y[gid] = best;
}

template <int BITS>
__global__ void __launch_bounds__(256) maxpool_byte_kernel(int n, int h, int w, int c, int k, int s, int oh, int ow,
                                                           const uint8_t *x, uint8_t *y)
{
    const int bytes_per_pix = c * BITS / 8;
    const long long total = static_cast<long long>(n) * oh * ow * bytes_per_pix;
    const long long gid = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (gid >= total) return;
    const int byte = static_cast<int>(gid % bytes_per_pix);
    const long long pix = gid / bytes_per_pix;
    const int ox = static_cast<int>(pix % ow);
    const int oy = static_cast<int>((pix / ow) % oh);
    const int b = static_cast<int>(pix / (static_cast<long long>(ow) * oh));
    constexpr int per = 8 / BITS;
    constexpr int mask = (1 << BITS) - 1;
    int best[per];
#pragma unroll
    for (int f = 0; f < per; ++f) best[f] = 0;
    for (int i = 0; i < k; ++i)
        for (int j = 0; j < k; ++j) {
            const long long src = ((static_cast<long long>(b) * h + oy * s + i) * w + ox * s + j) * bytes_per_pix + byte;
            const int t = x[src];
#pragma unroll
            for (int f = 0; f < per; ++f) best[f] = max(best[f], (t >> (f * BITS)) & mask);
        }
    int out = 0;
#pragma unroll
    for (int f = 0; f < per; ++f) out |= best[f] << (f * BITS);
    y[gid] = static_cast<uint8_t>(out);
}

}  // namespace

cudaError_t launch_maxpool(int n, int h, int w, int c, int k, int s, int bits, const uint8_t *x, uint8_t *y,
                           cudaStream_t st)
{
    const int oh = (h - k) / s + 1, ow = (w - k) / s + 1;
    const long long pix = static_cast<long long>(n) * oh * ow;
    if (pix == 0) return cudaSuccess;
    const int bytes_per_pix = c * bits / 8;
    const bool vec = bytes_per_pix % 16 == 0 && (reinterpret_cast<uintptr_t>(x) % 16) == 0 &&
                     (reinterpret_cast<uintptr_t>(y) % 16) == 0;
    if (vec) {
        const int vpp = bytes_per_pix / 16;
        const long long total = pix * vpp;
        const unsigned grid = static_cast<unsigned>((total + 255) / 256);
        const uint4 *xv = reinterpret_cast<const uint4 *>(x);
        uint4 *yv = reinterpret_cast<uint4 *>(y);
        if (bits == 8) maxpool_vec_kernel<8><<<grid, 256, 0, st>>>(n, h, w, vpp, k, s, oh, ow, xv, yv);
        else if (bits == 4) maxpool_vec_kernel<4><<<grid, 256, 0, st>>>(n, h, w, vpp, k, s, oh, ow, xv, yv);
        else maxpool_vec_kernel<2><<<grid, 256, 0, st>>>(n, h, w, vpp, k, s, oh, ow, xv, yv);
    } else {
        const long long total = pix * (c * bits / 8);
        const unsigned grid = static_cast<unsigned>((total + 255) / 256);
        if (bits == 8) maxpool_byte_kernel<8><<<grid, 256, 0, st>>>(n, h, w, c, k, s, oh, ow, x, y);
        else if (bits == 4) maxpool_byte_kernel<4><<<grid, 256, 0, st>>>(n, h, w, c, k, s, oh, ow, x, y);
        else maxpool_byte_kernel<2><<<grid, 256, 0, st>>>(n, h, w, c, k, s, oh, ow, x, y);
    }
    return cudaGetLastError();
}

}  // namespace qnn
