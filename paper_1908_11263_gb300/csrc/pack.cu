// Sub-byte packing and unpacking (Sec. IV-A, "Sub-byte Extensions"): Q-bit
// values stored 8/Q per byte, element e at bits [(e mod (8/Q)) * Q, +Q) of byte
// e / (8/Q).  One thread per packed byte.
#include <cstdint>

#include "internal.h"

namespace qnn {
namespace {

template <int BITS>
__global__ void __launch_bounds__(256) pack_kernel(const int8_t *src, uint8_t *dst, long long nbytes)
{
    const long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= nbytes) return;
    constexpr int per = 8 / BITS;
    int out = 0;
#pragma unroll
    for (int f = 0; f < per; ++f) out |= (src[i * per + f] & ((1 << BITS) - 1)) << (f * BITS);
    dst[i] = static_cast<uint8_t>(out);
}

template <int BITS>
__global__ void __launch_bounds__(256) unpack_kernel(const uint8_t *src, int8_t *dst, long long nbytes, int is_signed)
{
    const long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= nbytes) return;
    constexpr int per = 8 / BITS;
    const int byte = src[i];
#pragma unroll
    for (int f = 0; f < per; ++f) {
        int v = (byte >> (f * BITS)) & ((1 << BITS) - 1);
        if (is_signed && v >= (1 << (BITS - 1))) v -= (1 << BITS);
        dst[i * per + f] = static_cast<int8_t>(v);
    }
}

}  // namespace

cudaError_t launch_pack(const int8_t *src, uint8_t *dst, long long count, int bits, cudaStream_t st)
{
    const long long nbytes = count * bits / 8;
    if (nbytes == 0) return cudaSuccess;
    const unsigned grid = static_cast<unsigned>((nbytes + 255) / 256);
    if (bits == 8) pack_kernel<8><<<grid, 256, 0, st>>>(src, dst, nbytes);
    else if (bits == 4) pack_kernel<4><<<grid, 256, 0, st>>>(src, dst, nbytes);
    else pack_kernel<2><<<grid, 256, 0, st>>>(src, dst, nbytes);
    return cudaGetLastError();
}

cudaError_t launch_unpack(const uint8_t *src, int8_t *dst, long long count, int bits, int is_signed, cudaStream_t st)
{
    const long long nbytes = count * bits / 8;
    if (nbytes == 0) return cudaSuccess;
    const unsigned grid = static_cast<unsigned>((nbytes + 255) / 256);
    if (bits == 8) unpack_kernel<8><<<grid, 256, 0, st>>>(src, dst, nbytes, is_signed);
    else if (bits == 4) unpack_kernel<4><<<grid, 256, 0, st>>>(src, dst, nbytes, is_signed);
    else unpack_kernel<2><<<grid, 256, 0, st>>>(src, dst, nbytes, is_signed);
    return cudaGetLastError();
}

}  // namespace qnn
