// INT-1 convolution (Sec. III-A, Eq. 5; binary kernel of Sec. IV-A).  Values
// +1 / -1 are bits 1 / 0, eight per byte (element e at bit e mod 8 of byte
// e / 8).  The accumulator counts the ones of W xnor X over the window
// positions inside the image (padding contributes nothing), and the output
// bit is 1 when the channel's threshold does not exceed it.
//
// One thread per output pixel: a warp covers 32 consecutive pixels, so its
// input words are coalesced, and every lane reads the same weight words (a
// broadcast).  Output channels go 32 at a time with the counts in registers;
// each input word is used for all 32 before the next is loaded.
#include <cstdint>

#include "internal.h"

namespace qnn {
namespace {

constexpr int kChanChunk = 32;

// UNIT: uint32_t when C is a multiple of 32, else uint8_t (C is a multiple of 8).
template <typename UNIT>
__global__ void __launch_bounds__(256) conv_binary_kernel(ConvShape s, const uint8_t *x, const uint8_t *w,
                                                          const int32_t *thr, uint8_t *y)
{
    const long long npix = static_cast<long long>(s.n) * s.oh * s.ow;
    const long long pix = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (pix >= npix) return;
    const int ox = static_cast<int>(pix % s.ow);
    const int oy = static_cast<int>((pix / s.ow) % s.oh);
    const int b = static_cast<int>(pix / (static_cast<long long>(s.ow) * s.oh));
    constexpr int kBitsPerUnit = 8 * sizeof(UNIT);
    const int units = s.c / kBitsPerUnit;  // units per tap and pixel
    const int taps = s.kh * s.kw;
    const UNIT *xu = reinterpret_cast<const UNIT *>(x);
    const UNIT *wu = reinterpret_cast<const UNIT *>(w);
    for (int o0 = 0; o0 < s.m; o0 += kChanChunk) {
        int acc[kChanChunk];
#pragma unroll
        for (int k = 0; k < kChanChunk; ++k) acc[k] = 0;
        for (int i = 0; i < s.kh; ++i) {
            const int iy = oy * s.sh - s.ph + i;
            if (iy < 0 || iy >= s.h) continue;
            for (int j = 0; j < s.kw; ++j) {
                const int ix = ox * s.sw - s.pw + j;
                if (ix < 0 || ix >= s.w) continue;
                const long long xo = ((static_cast<long long>(b) * s.h + iy) * s.w + ix) * units;
                const int tap = i * s.kw + j;
                for (int u = 0; u < units; ++u) {
                    const uint32_t xv = __ldg(xu + xo + u);
#pragma unroll
                    for (int k = 0; k < kChanChunk; ++k) {
                        if (o0 + k < s.m) {
                            const uint32_t wv = __ldg(wu + (static_cast<long long>(o0 + k) * taps + tap) * units + u);
                            const uint32_t match = ~(xv ^ wv) & (kBitsPerUnit == 32 ? 0xffffffffu : 0xffu);
                            acc[k] += __popc(match);
                        }
                    }
                }
            }
        }
        // thresholds and bit packing: 8 channels per output byte
        uint8_t *yp = y + pix * (s.m / 8) + o0 / 8;
#pragma unroll
        for (int byte = 0; byte < kChanChunk / 8; ++byte) {
            if (o0 + 8 * byte >= s.m) break;
            uint32_t bits = 0;
#pragma unroll
            for (int q = 0; q < 8; ++q) bits |= (thr[o0 + 8 * byte + q] <= acc[8 * byte + q] ? 1u : 0u) << q;
            yp[byte] = static_cast<uint8_t>(bits);
        }
    }
}

// Weights staged once per block in shared memory as [tap * units + u][m4]
// words (m4 = m rounded up to 4, zero-filled), so one broadcast 128-bit load
// serves four channels.  32-bit words (C a multiple of 32).
constexpr int kSmemWeightsMax = 48 * 1024;

__global__ void __launch_bounds__(256) conv_binary_smem_kernel(ConvShape s, const uint32_t *x, const uint32_t *w,
                                                               const int32_t *thr, uint8_t *y)
{
    extern __shared__ uint4 wsh4[];
    uint32_t *wsh = reinterpret_cast<uint32_t *>(wsh4);
    const int units = s.c / 32, taps = s.kh * s.kw, m4 = (s.m + 3) & ~3;
    const int rows = taps * units;
    for (int i = threadIdx.x; i < rows * m4; i += blockDim.x) {
        const int tu = i / m4, o = i - tu * m4;
        wsh[i] = o < s.m ? __ldg(w + static_cast<long long>(o) * rows + tu) : 0u;  // w is [o][tap][u]
    }
    __syncthreads();
    const long long npix = static_cast<long long>(s.n) * s.oh * s.ow;
    const long long pix = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (pix >= npix) return;
    const int ox = static_cast<int>(pix % s.ow);
    const int oy = static_cast<int>((pix / s.ow) % s.oh);
    const int b = static_cast<int>(pix / (static_cast<long long>(s.ow) * s.oh));
    for (int o0 = 0; o0 < s.m; o0 += kChanChunk) {
        int acc[kChanChunk];
#pragma unroll
        for (int k = 0; k < kChanChunk; ++k) acc[k] = 0;
        for (int i = 0; i < s.kh; ++i) {
            const int iy = oy * s.sh - s.ph + i;
            if (iy < 0 || iy >= s.h) continue;
            for (int j = 0; j < s.kw; ++j) {
                const int ix = ox * s.sw - s.pw + j;
                if (ix < 0 || ix >= s.w) continue;
                const long long xo = ((static_cast<long long>(b) * s.h + iy) * s.w + ix) * units;
                const int tap = i * s.kw + j;
                for (int u = 0; u < units; ++u) {
                    const uint32_t xv = __ldg(x + xo + u);
                    const uint4 *wr = reinterpret_cast<const uint4 *>(wsh + (tap * units + u) * m4 + o0);
#pragma unroll
                    for (int q = 0; q < kChanChunk / 4; ++q) {
                        if (o0 + 4 * q < s.m) {
                            const uint4 wv = wr[q];
                            acc[4 * q] += __popc(~(xv ^ wv.x));
                            acc[4 * q + 1] += __popc(~(xv ^ wv.y));
                            acc[4 * q + 2] += __popc(~(xv ^ wv.z));
                            acc[4 * q + 3] += __popc(~(xv ^ wv.w));
                        }
                    }
                }
            }
        }
        uint8_t *yp = y + pix * (s.m / 8) + o0 / 8;
#pragma unroll
        for (int byte = 0; byte < kChanChunk / 8; ++byte) {
            if (o0 + 8 * byte >= s.m) break;
            uint32_t bits = 0;
#pragma unroll
            for (int q = 0; q < 8; ++q) bits |= (thr[o0 + 8 * byte + q] <= acc[8 * byte + q] ? 1u : 0u) << q;
            yp[byte] = static_cast<uint8_t>(bits);
        }
    }
}

}  // namespace

cudaError_t launch_conv_binary(const ConvShape &s, const uint8_t *x, const uint8_t *w, const int32_t *thr, uint8_t *y,
                               cudaStream_t st)
{
    const long long npix = static_cast<long long>(s.n) * s.oh * s.ow;
    if (npix == 0) return cudaSuccess;
    const unsigned grid = static_cast<unsigned>((npix + 255) / 256);
    const bool words = s.c % 32 == 0 && (reinterpret_cast<uintptr_t>(x) % 4) == 0 &&
                       (reinterpret_cast<uintptr_t>(w) % 4) == 0;
    const size_t smem = static_cast<size_t>(s.kh) * s.kw * (s.c / 32) * ((s.m + 3) & ~3) * 4;
    if (words && smem <= static_cast<size_t>(kSmemWeightsMax))
        conv_binary_smem_kernel<<<grid, 256, smem, st>>>(s, reinterpret_cast<const uint32_t *>(x),
                                                         reinterpret_cast<const uint32_t *>(w), thr, y);
    else if (words) conv_binary_kernel<uint32_t><<<grid, 256, 0, st>>>(s, x, w, thr, y);
    else conv_binary_kernel<uint8_t><<<grid, 256, 0, st>>>(s, x, w, thr, y);
    return cudaGetLastError();
}

}  // namespace qnn
