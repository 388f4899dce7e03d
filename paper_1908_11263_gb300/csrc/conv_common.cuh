// Device helpers shared by the tensor-core convolution kernels (conv_tc.cu,
// conv_win.cu): exact staging encodings of packed activations, the compression
// step of Sec. III-A fused with Q-bit packing (Sec. IV-A), and the arithmetic
// that proves per channel which compression form is exact.  sm_103a only.
#pragma once

#include <cuda_fp16.h>

#include <cstdint>

#include "device.cuh"

namespace qnn {
namespace {

constexpr uint32_t kMagic = 0x4B400000u;  // bits of 1.5 * 2^23: the accumulator pre-load

// Division by a runtime constant d in [1, 2^32) for 32-bit numerators:
// q = floor(n * m / 2^64) with m = ceil(2^64 / d).  Exact: m * d = 2^64 + e with
// 0 <= e < d, so n * m / 2^64 = n / d + n * e / (d * 2^64), and the second term
// is below 1/d for n < 2^32, too small to carry past the next integer.  m = 0
// stands for d = 1.
struct FastDiv {
    unsigned long long m;
    uint32_t d;
};

FastDiv make_fastdiv(uint32_t d)
{
    FastDiv f;
    f.d = d;
    f.m = d <= 1 ? 0ull : (~0ull / d) + 1ull;
    return f;
}

__device__ __forceinline__ int fdiv(int n, const FastDiv &f)
{
    return f.m == 0ull ? n : static_cast<int>(__umul64hi(static_cast<unsigned long long>(n), f.m));
}

// Per-channel compression constants (two records per channel, see the prep kernel).
//   rec0 = {lam2, kappa, shift, mode}   rec1 = {beta, ulo, uhi, lambda}
enum { kModeWide = 0, kModeClamp = 1, kModeDirect = 2, kModeThreshold = 3 };
// Staircase compression: each channel's 2^Q - 1 thresholds, stored kThrStride
// int32 apart in the workspace and in shared memory.
constexpr int kThrStride = 16;

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel)
{
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

__device__ __forceinline__ uint32_t hsub2(uint32_t a, uint32_t b)
{
    uint32_t d;
    asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

// Encoded activation 0 (padding and channels beyond c).
template <int BITS>
__device__ __forceinline__ uint32_t pad_half2()
{
    return BITS == 8 ? 0xD800D800u /* -128.0 */ : 0x64006400u /* 1024.0 */;
}

// 8 unsigned bytes -> 8 fp16 (x - 128), natural channel order.
__device__ __forceinline__ uint4 cvt_u8x8(uint2 v)
{
    const uint32_t k64 = 0x64646464u, k1152 = 0x64806480u;  // fp16 1152 = 1024 + 128
    uint4 r;
    r.x = hsub2(prmt(v.x, k64, 0x4140), k1152);
    r.y = hsub2(prmt(v.x, k64, 0x4342), k1152);
    r.z = hsub2(prmt(v.y, k64, 0x4140), k1152);
    r.w = hsub2(prmt(v.y, k64, 0x4342), k1152);
    return r;
}

// 8 nibbles (one 32-bit word) -> 8 fp16 (x + 1024); slot s holds channel {0,4,1,5,2,6,3,7}[s].
__device__ __forceinline__ uint4 cvt_u4x8(uint32_t v)
{
    const uint32_t m = 0x000F000Fu, k = 0x64006400u;
    uint4 r;
    r.x = (v & m) | k;
    r.y = ((v >> 4) & m) | k;
    r.z = ((v >> 8) & m) | k;
    r.w = ((v >> 12) & m) | k;
    return r;
}

// 8 crumbs (16 bits) -> 8 fp16 (x + 1024); slot s holds channel {0,4,1,5,2,6,3,7}[s].
__device__ __forceinline__ uint4 cvt_u2x8(uint32_t v16)
{
    const uint32_t t = (v16 & 0xFFu) | ((v16 & 0xFF00u) << 8);
    const uint32_t m = 0x00030003u, k = 0x64006400u;
    uint4 r;
    r.x = (t & m) | k;
    r.y = ((t >> 2) & m) | k;
    r.z = ((t >> 4) & m) | k;
    r.w = ((t >> 6) & m) | k;
    return r;
}

__device__ __forceinline__ void sts128(uint32_t addr, uint4 v)
{
    asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w));
}

// Predicated 128-bit shared store (no branch around it).
__device__ __forceinline__ void sts128_if(bool pred, uint32_t addr, uint4 v)
{
    asm volatile(
        "{\n\t.reg .pred q;\n\t"
        "setp.ne.b32 q, %5, 0;\n\t"
        "@q st.shared.v4.b32 [%0], {%1,%2,%3,%4};\n\t}" ::"r"(addr),
        "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(static_cast<int>(pred)));
}

// e4m3 codes of four 4-bit values v0..v3 (selector nibbles, bits 0-15): value
// v goes to byte k.  Two 8-entry lookups: prmt picks byte v & 7 of a table,
// and a selector nibble with bit 3 set yields that byte's sign, 0 here, so
// each lookup answers for its own half of 0..15 and zero for the other.  The
// tables hold e4m3(v) = 2^(E-7) * (1 + M/8) for v = 0..7 and 8..15, all exact.
__device__ __forceinline__ uint32_t e4m3x4(uint32_t sel)
{
    return prmt(0x44403800u, 0x4E4C4A48u, sel) | prmt(0x53525150u, 0x57565554u, sel ^ 0x8888u);
}

// 16 unsigned INT-4 (one 8-byte load) or INT-2 (one 4-byte load) activations
// -> 16 e4m3 bytes.  INT-4 keeps the channel order; INT-2 yields channels
// {0,2,4,6}, {1,3,5,7}, {8,10,12,14}, {9,11,13,15} in its four words (the
// filters are laid out to match).
template <int BITS>
__device__ __forceinline__ uint4 cvt_raw_f8(const uint8_t *p)
{
    uint4 r;
    if (BITS == 4) {
        const uint2 v = *reinterpret_cast<const uint2 *>(p);
        r = make_uint4(e4m3x4(v.x), e4m3x4(v.x >> 16), e4m3x4(v.y), e4m3x4(v.y >> 16));
    } else {
        const uint32_t v = *reinterpret_cast<const uint32_t *>(p);
        const uint32_t ev = v & 0x33333333u, od = (v >> 2) & 0x33333333u;  // crumbs 2k and 2k+1 as nibbles
        r = make_uint4(e4m3x4(ev), e4m3x4(od), e4m3x4(ev >> 16), e4m3x4(od >> 16));
    }
    return r;
}

template <int BITS>
__device__ __forceinline__ uint4 cvt_raw(const uint8_t *p)
{
    if (BITS == 8) return cvt_u8x8(*reinterpret_cast<const uint2 *>(p));
    if (BITS == 4) return cvt_u4x8(*reinterpret_cast<const uint32_t *>(p));
    return cvt_u2x8(*reinterpret_cast<const uint16_t *>(p));
}

// Compression of one integer sum u = acc + bias in 64-bit arithmetic.
__device__ __noinline__ uint32_t compress64(int32_t u, int32_t kappa, int32_t lambda, int32_t shift, uint32_t top)
{
    long long t = static_cast<long long>(u) * kappa + lambda;
    t >>= shift;
    return t < 0 ? 0u : (t > static_cast<long long>(top) ? top : static_cast<uint32_t>(t));
}

// Channels whose constants need more than the direct form: raw chunk sum s ->
// output, by the clamped 32-bit form, the 64-bit routine or the staircase
// (Eq. 4: the number of the channel's thresholds that do not exceed
// acc = s + beta; in that mode rec0.x is the shared-memory byte offset of the
// channel's thresholds, set when the records are staged).
__device__ __noinline__ uint32_t compress_slow(uint32_t s, int4 r0, int4 r1, uint32_t top)
{
    const int32_t u = static_cast<int32_t>(s + static_cast<uint32_t>(r1.x));
    if (r0.w == kModeThreshold) {
        extern __shared__ __align__(128) uint8_t smem[];
        const int32_t *tau = reinterpret_cast<const int32_t *>(smem + r0.x);
        uint32_t y = 0;
        for (uint32_t k = 0; k < top; ++k) y += tau[k] <= u ? 1u : 0u;
        return y;
    }
    if (r0.w == kModeClamp) {
        const int32_t uc = min(max(u, r1.y), r1.z);
        const int32_t t = (uc * r0.y + r1.w) >> r0.z;
        return static_cast<uint32_t>(min(max(t, 0), static_cast<int32_t>(top)));
    }
    return compress64(u, r0.y, r1.w, r0.z, top);
}

// Saturating pack of two results (cvt.pack.sat): returns
// (upper << 2Q) | (clip(hi) << Q) | clip(lo) with clip to [0, 2^Q - 1], the
// clip of the compression step (Sec. III-A) fused with the Q-bit packing of
// Sec. IV-A.
template <int BITS>
__device__ __forceinline__ uint32_t pack2_sat(int hi, int lo, uint32_t upper)
{
    uint32_t d;
    if (BITS == 8) asm("cvt.pack.sat.u8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(hi), "r"(lo), "r"(upper));
    else if (BITS == 4) asm("cvt.pack.sat.u4.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(hi), "r"(lo), "r"(upper));
    else asm("cvt.pack.sat.u2.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(hi), "r"(lo), "r"(upper));
    return d;
}

// Compression (Sec. III-A) of G raw sums of one pixel, Q-bit packing (Sec.
// IV-A) and store of the channels below m.  Direct channels (the common case)
// compute ((s * kappa + lam2) mod 2^32) >> shift and clip it: the prep kernel
// has proved that (acc + bias) * kappa + lambda stays inside int32 for every
// accumulator the layer can produce, and folded bias, the staging offset and
// the accumulator pre-load into lam2, so the wrapped 32-bit value is exact.
template <int BITS, int G>
__device__ __forceinline__ void compress_pack(const uint32_t *s, const int4 *rec0, const int4 *rec1, bool direct,
                                              int m_first, uint32_t (&packed)[(G * BITS + 31) / 32])
{
    int y[G];
    if (direct) {
#pragma unroll
        for (int k = 0; k < G; ++k) {
            const int4 r0 = rec0[m_first + k];
            y[k] = static_cast<int32_t>(s[k] * static_cast<uint32_t>(r0.y) + static_cast<uint32_t>(r0.x)) >> r0.z;
        }
    } else {
#pragma unroll
        for (int k = 0; k < G; ++k)
            y[k] = static_cast<int>(compress_slow(s[k], rec0[m_first + k], rec1[m_first + k], (1u << BITS) - 1u));
    }
    constexpr int kPer = 32 / BITS;                   // results per 32-bit word
    constexpr int kWords = (G * BITS + 31) / 32;
#pragma unroll
    for (int wd = 0; wd < kWords; ++wd) {
        uint32_t t = 0;
#pragma unroll
        for (int k = kPer - 2; k >= 0; k -= 2) {  // highest pair first; it ends in the top bits
            const int e = wd * kPer + k;
            if (e < G) t = pack2_sat<BITS>(y[e + 1], y[e], t);
        }
        packed[wd] = t;
    }
}

// Stores G packed Q-bit outputs (fewer when `valid` < G, at the end of M).
template <int BITS, int G>
__device__ __forceinline__ void store_packed(const uint32_t (&packed)[(G * BITS + 31) / 32], int valid, uint8_t *dst)
{
    constexpr int kWords = (G * BITS + 31) / 32;
    constexpr int kBytes = G * BITS / 8;
    if (valid >= G && (reinterpret_cast<uintptr_t>(dst) % (kBytes < 16 ? kBytes : 16)) == 0) {
        if (kBytes >= 16) {
#pragma unroll
            for (int q = 0; q < kBytes / 16; ++q)
                reinterpret_cast<uint4 *>(dst)[q] =
                    make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2], packed[4 * q + 3]);
        }
        else if (kBytes == 8) *reinterpret_cast<uint2 *>(dst) = make_uint2(packed[0], packed[kWords > 1 ? 1 : 0]);
        else if (kBytes == 4) *reinterpret_cast<uint32_t *>(dst) = packed[0];
        else if (kBytes == 2) *reinterpret_cast<uint16_t *>(dst) = static_cast<uint16_t>(packed[0]);
        else *dst = static_cast<uint8_t>(packed[0]);
    } else {
        const int nbytes = min(valid, G) * BITS / 8;
#pragma unroll
        for (int b = 0; b < kBytes; ++b)
            if (b < nbytes) dst[b] = static_cast<uint8_t>(packed[b / 4] >> (8 * (b % 4)));
    }
}

template <int BITS, int G>
__device__ __forceinline__ void compress_store(const uint32_t *s, const int4 *rec0, const int4 *rec1, bool direct,
                                               int m_first, int valid, uint8_t *dst)
{
    uint32_t packed[(G * BITS + 31) / 32];
    compress_pack<BITS, G>(s, rec0, rec1, direct, m_first, packed);
    store_packed<BITS, G>(packed, valid, dst);
}

__device__ __forceinline__ long long floor_div(long long a, long long b)
{
    long long q = a / b;
    if ((a % b != 0) && ((a < 0) != (b < 0))) --q;
    return q;
}

__device__ __forceinline__ long long ceil_div(long long a, long long b) { return -floor_div(-a, b); }

__device__ __forceinline__ bool in_i32(long long v) { return v >= INT32_MIN && v <= INT32_MAX; }

// For y(u) = clip(floor((u*kappa + lambda) / 2^s), 0, top): an interval [ulo, uhi]
// outside which y is constant (0 or top, whichever side), chosen so that
// clamping u into it never changes y.  Returns true when u*kappa + lambda stays
// inside int32 for every u in the interval (the clamped 32-bit form is exact).
__device__ bool saturation_bounds(long long kappa, long long lambda, int s, long long top, long long *ulo,
                                  long long *uhi)
{
    const long long one = 1ll << s;
    if (kappa > 0) {
        *ulo = ceil_div(one - lambda, kappa) - 1;    // y(u) = 0 for every u <= ulo
        *uhi = ceil_div(top * one - lambda, kappa);  // y(u) = top for every u >= uhi
    } else if (kappa < 0) {
        *ulo = floor_div(top * one - lambda, kappa);  // y(u) = top for every u <= ulo
        *uhi = floor_div(one - lambda, kappa) + 1;    // y(u) = 0 for every u >= uhi
    } else {
        *ulo = 0;
        *uhi = 0;
    }
    if (*ulo < INT32_MIN) *ulo = INT32_MIN;
    if (*uhi > INT32_MAX) *uhi = INT32_MAX;
    if (*ulo > *uhi) *ulo = *uhi;
    return in_i32(*ulo * kappa + lambda) && in_i32(*uhi * kappa + lambda);
}

// e4m3 code of an integer with |v| <= 15 (exact): sign, exponent e + 7 for
// |v| in [2^e, 2^(e+1)), three fraction bits.
__device__ __forceinline__ uint8_t e4m3_of_int(int v)
{
    if (v == 0) return 0;
    const uint32_t sgn = v < 0 ? 0x80u : 0u;
    const uint32_t mag = static_cast<uint32_t>(v < 0 ? -v : v);
    const int e = 31 - __clz(static_cast<int>(mag));
    const uint32_t frac = ((mag << 3) >> e) & 7u;
    return static_cast<uint8_t>(sgn | (static_cast<uint32_t>(e + 7) << 3) | frac);
}

}  // namespace
}  // namespace qnn
