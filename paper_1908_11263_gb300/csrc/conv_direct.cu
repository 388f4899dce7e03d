// Quantized HWC convolution on the CUDA cores (any stride and padding).
//
// Same computation as the tensor-core kernel (Sec. III-B, Eq. 6, with the
// compression of Sec. III-A), written as the direct sum: one thread computes 8
// consecutive output channels of one output pixel, accumulating exact int32
// products.  For INT-8 data with c % 4 == 0 the inner loop uses dp4a.u32.s32
// (four u8 x s8 products per instruction, the GPU counterpart of the paper's
// sdotp4); other layouts unpack element by element.  Used for strides other
// than 1 and as an independent second GPU path in the tests.
#include <cstdint>

#include "device.cuh"
#include "internal.h"

namespace qnn {
namespace {

constexpr int kOutPerThread = 8;

__device__ __forceinline__ int dp4a_us(uint32_t a, uint32_t b, int c)
{
    int d;
    asm("dp4a.u32.s32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}

template <int BITS>
__device__ __forceinline__ int field_u(const uint8_t *base, long long e)
{
    if (BITS == 8) return base[e];
    constexpr int per = 8 / BITS;
    return (base[e / per] >> ((e % per) * BITS)) & ((1 << BITS) - 1);
}

template <int BITS>
__device__ __forceinline__ int field_s(const uint8_t *base, long long e)
{
    const int f = field_u<BITS>(base, e);
    return f >= (1 << (BITS - 1)) ? f - (1 << BITS) : f;
}

template <int BITS, bool DP4A>
__global__ void __launch_bounds__(128) conv_direct_kernel(ConvShape s, ConvParams p)
{
    const long long npix = static_cast<long long>(s.n) * s.oh * s.ow;
    const int groups = (s.m + kOutPerThread - 1) / kOutPerThread;
    const long long gid = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (gid >= npix * groups) return;
    const int grp = static_cast<int>(gid % groups);
    const long long pix = gid / groups;
    const int ox = static_cast<int>(pix % s.ow);
    const int oy = static_cast<int>((pix / s.ow) % s.oh);
    const int b = static_cast<int>(pix / (static_cast<long long>(s.ow) * s.oh));
    const int o0 = grp * kOutPerThread;
    const int nout = min(kOutPerThread, s.m - o0);

    int acc[kOutPerThread];
#pragma unroll
    for (int k = 0; k < kOutPerThread; ++k) acc[k] = 0;

    for (int i = 0; i < s.kh; ++i) {
        const int iy = oy * s.sh - s.ph + i;
        if (iy < 0 || iy >= s.h) continue;
        for (int j = 0; j < s.kw; ++j) {
            const int ix = ox * s.sw - s.pw + j;
            if (ix < 0 || ix >= s.w) continue;
            const long long xe = ((static_cast<long long>(b) * s.h + iy) * s.w + ix) * s.c;
            const long long we = (static_cast<long long>(i) * s.kw + j) * s.c;
            const long long wstride = static_cast<long long>(s.kh) * s.kw * s.c;
            if (DP4A) {
                const uint32_t *xw = reinterpret_cast<const uint32_t *>(p.x + xe);
                for (int c4 = 0; c4 < s.c / 4; ++c4) {
                    const uint32_t xv = __ldg(xw + c4);
#pragma unroll
                    for (int k = 0; k < kOutPerThread; ++k) {
                        if (k < nout) {
                            const uint32_t wv =
                                __ldg(reinterpret_cast<const uint32_t *>(p.w + (o0 + k) * wstride + we) + c4);
                            acc[k] = dp4a_us(xv, wv, acc[k]);
                        }
                    }
                }
            } else {
                for (int ch = 0; ch < s.c; ++ch) {
                    const int xv = field_u<BITS>(p.x, xe + ch);
#pragma unroll
                    for (int k = 0; k < kOutPerThread; ++k)
                        if (k < nout) acc[k] += xv * field_s<BITS>(p.w, (o0 + k) * wstride + we + ch);
                }
            }
        }
    }

    // compression (Sec. III-A) and packing of the 8 outputs (Sec. IV-A)
    const long long top = (1 << BITS) - 1;
    const long long ye = pix * s.m + o0;  // element index of the first output
#pragma unroll
    for (int k = 0; k < kOutPerThread; ++k) {
        if (k >= nout) break;
        const int o = o0 + k;
        int yv;
        if (p.thresholds) {  // staircase (Eq. 4): thresholds that do not exceed the accumulator
            const int32_t *tau = p.thresholds + static_cast<long long>(o) * top;
            yv = 0;
            for (int q = 0; q < top; ++q) yv += tau[q] <= acc[k] ? 1 : 0;
        } else {
            const int32_t u = acc[k] + (p.bias ? p.bias[o] : 0);
            long long t = static_cast<long long>(u) * p.kappa[o] + p.lambda[o];
            t >>= (p.shifts ? p.shifts[o] : p.shift);
            yv = static_cast<int>(t < 0 ? 0 : (t > top ? top : t));
        }
        if (BITS == 8) {
            p.y[ye + k] = static_cast<uint8_t>(yv);
        } else {
            // this thread owns whole bytes: o0 is a multiple of 8 and m of 8/Q
            constexpr int per = 8 / BITS;
            const long long e = ye + k;
            uint8_t *dst = p.y + e / per;
            const int pos = static_cast<int>(e % per) * BITS;
            if (pos == 0) *dst = static_cast<uint8_t>(yv);
            else *dst = static_cast<uint8_t>(*dst | (yv << pos));
        }
    }
}

template <int BITS>
cudaError_t launch_bits(const ConvShape &s, const ConvParams &p, cudaStream_t st)
{
    const long long npix = static_cast<long long>(s.n) * s.oh * s.ow;
    const long long work = npix * ((s.m + kOutPerThread - 1) / kOutPerThread);
    if (work == 0) return cudaSuccess;
    const unsigned grid = static_cast<unsigned>((work + 127) / 128);
    if (BITS == 8 && s.c % 4 == 0)
        conv_direct_kernel<8, true><<<grid, 128, 0, st>>>(s, p);
    else
        conv_direct_kernel<BITS, false><<<grid, 128, 0, st>>>(s, p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_conv_direct(const ConvShape &s, const ConvParams &p, cudaStream_t st)
{
    switch (s.bits) {
        case 8: return launch_bits<8>(s, p, st);
        case 4: return launch_bits<4>(s, p, st);
        default: return launch_bits<2>(s, p, st);
    }
}

}  // namespace qnn
