// Quantized HWC convolution on the sm_103a tensor cores in one launch: the
// window kernel.  Included by conv_win_q8.cu, conv_win_q4.cu and conv_win_q2.cu,
// one bit width each, so the three compile in parallel.
//
// What it computes (Sec. III-B, Eq. 6; Sec. III-A): for every output pixel p
// and channel o,
//   acc = dot(W(o), im2col(p))                       exact integer, int32
//   y   = clip(floor(((acc + bias_o) * kappa_o + lambda_o) / 2^shift_o), 0, 2^Q - 1)
// or, with thresholds, the staircase of Eq. 4; optionally followed by the 2x2
// stride-2 max-pool of Sec. IV-A.
//
// Tiles.  A tile is S strips side by side, each 16 output rows x 8 output
// columns; the tile's input is staged once as a padded window of
// (16 + kh - 1) rows x (8S + kw - 1) pixels.  Strip s of tap (i, j) is the
// 128 x K operand that starts at window position i * sp + j + 8 s: its sixteen
// 8-row core-matrix groups are the sixteen output rows, sp positions apart.
// One shared-memory descriptor per MMA, no im2col buffer and no shifted
// copies (Eq. 7: neighbouring output pixels read neighbouring window pixels).
//
// Exactness on fp16 / e4m3 tensor cores (there is no integer tcgen05 MMA on
// this GPU).  INT-8 activations are staged as x - 128 in fp16, INT-4 / INT-2
// as themselves in e4m3; weights as themselves; all exact.  Every accumulator
// is pre-loaded with 1.5 * 2^23, so while the partial sums of a chunk stay
// within 2^22 of it every one is an integer that fp32 holds exactly; the bit
// pattern minus the pre-load is the chunk's integer sum.  The kernel derives
// the number of chunks from the filters themselves: the fewest contiguous tap
// ranges for which max|staged x| * sum|w| over the range stays within 2^22 for
// every output channel (the worst case over all filters is the planner's
// nch_max, always valid).
//
// Filters in the kernel.  The epilogue warps start by reading the packed
// filters and per-channel constants and writing the B operand (K-major
// core matrices) and the compression records into shared memory, while the
// loader and converter warps stage the first windows.  So one qconv_hwc call
// is one launch and needs no workspace.
//
// Warp roles (one persistent CTA per SM, 14 warps):
//   warps 0-3   converters: raw window -> staged operand, every position
//   warps 4-11  filter preparation, then epilogue: warp w reads TMEM lane
//               quarter w % 4 and one half of the output channels; sums the
//               chunks, compresses, packs at Q bits and stores
//   warp 12     MMA issue (converged warp, elected lane)
//   warp 13     bulk copies of the input rows of each window
// Every wait is bounded; on a timeout the kernel records QNN_ETIMEOUT in the
// status word, stops, lets its copies and MMAs drain and frees TMEM.
#pragma once

#include "conv_common.cuh"
#include "device.cuh"
#include "internal.h"

namespace qnn {
namespace win {

constexpr int kConvWarps = 4, kEpiWarps = 8;
constexpr int kEpiWarp0 = 4, kMmaWarp = 12, kLoadWarp = 13;
constexpr int kWarps = 14;
constexpr int kThreads = kWarps * 32;
constexpr int kRows = 16, kCols = 8;  // output rows and columns of one strip
constexpr int kMaxTaps = 64;
constexpr int kMaxSlots = 4;          // accumulator slots in TMEM
constexpr int kMaxStages = 4;         // raw windows / staged windows in flight
constexpr int kMaxKP = 5;             // window positions per converter thread and K-chunk plane
constexpr int kSmemLimit = 232448;    // 227 KB opt-in dynamic shared memory per block

// Shared-memory words after the barriers: the TMEM base, the chunk count the
// filters allow, the accumulator slot count and width, the chunk-mask vote.
struct Misc {
    uint32_t tmem;
    uint32_t nch;
    uint32_t nslots;
    uint32_t slot_cols;
    uint32_t mask;
    uint32_t pad[3];
};

struct WinArgs {
    const uint8_t *x;
    uint8_t *y;
    const uint8_t *w;        // packed filters [m][kh][kw][c]
    const int32_t *bias;     // [m] or null
    const int16_t *kappa;    // [m]
    const int32_t *lambda;   // [m]
    const uint8_t *shifts;   // [m] or null
    const int32_t *thr;      // [m][2^Q - 1] (staircase compression) or null
    int shift;
    int n, h, w_, c, m, kh, kw, ph, pw, oh, ow;
    int c_pad, groups, taps, ksteps, s, sp, wh, npos;
    int cb;                  // packed bytes per input pixel
    int full_rows;
    int tiles_x, tiles_per_img, total_tiles;
    FastDiv fd_tpi, fd_tx, fd_sp;
    int raw_stages, a_stages, nch_max;
    uint32_t raw_row_bytes, raw_bytes, chunk_stride, stage_bytes;
    uint32_t off_b, off_a, off_raw, off_rec, off_thr, off_tap, off_bar;
    int pool, pool_oh, pool_ow;
    int *status;
    uint32_t tap_a16[kMaxTaps];  // per tap (i, j): window position i * sp + j
};

// Tile t: image, first output row and column, window origin in the input.
struct Geo {
    int img, oy0, ox0, iy0, ix0;
};

__device__ __forceinline__ Geo geo_of(const WinArgs &a, int t)
{
    Geo g;
    g.img = fdiv(t, a.fd_tpi);
    const int ti = t - g.img * a.tiles_per_img;
    const int ty = fdiv(ti, a.fd_tx);
    g.oy0 = ty * kRows;
    g.ox0 = (ti - ty * a.tiles_x) * (kCols * a.s);
    g.iy0 = g.oy0 - a.ph;
    g.ix0 = g.ox0 - a.pw;
    return g;
}

// Window rows [r_lo, r_hi) and columns [c_lo, c_hi) that lie inside the image.
__device__ __forceinline__ int row_lo(const WinArgs &a, const Geo &g) { return min(a.wh, max(0, -g.iy0)); }
__device__ __forceinline__ int row_hi(const WinArgs &a, const Geo &g)
{
    return max(row_lo(a, g), min(a.wh, a.h - g.iy0));
}
__device__ __forceinline__ int col_lo(const WinArgs &a, const Geo &g) { return min(a.sp, max(0, -g.ix0)); }
__device__ __forceinline__ int col_hi(const WinArgs &a, const Geo &g)
{
    return max(col_lo(a, g), min(a.sp, a.w_ - g.ix0));
}

// ---------------------------------------------------------------- loader (warp 13)

// The input rows of each tile's window: one bulk copy when windows span whole
// image rows, else one per row (lanes issue them in parallel).
__device__ __forceinline__ void loader_role(const WinArgs &a, uint8_t *smem, uint64_t *raw_full, uint64_t *raw_empty)
{
    const int lane = threadIdx.x & 31;
    int rs = 0, issued = 0;
    uint32_t ph = 0;
    for (int t = blockIdx.x; t < a.total_tiles; t += gridDim.x) {
        const Geo g = geo_of(a, t);
        const int r0 = row_lo(a, g), r1 = row_hi(a, g);
        const int c0 = col_lo(a, g), c1 = col_hi(a, g);
        if (!mbar_wait_warp(&raw_empty[rs], ph ^ 1u, a.status)) break;
        uint8_t *dst = smem + a.off_raw + rs * a.raw_bytes;
        const int rows = r1 - r0;
        if (a.full_rows) {
            const uint32_t bytes = static_cast<uint32_t>(rows) * a.raw_row_bytes;
            if (lane == 0) {
                mbar_arrive_expect_tx(&raw_full[rs], bytes);
                const uint8_t *src = a.x + (static_cast<long long>(g.img) * a.h + (g.iy0 + r0)) * a.raw_row_bytes;
                for (uint32_t off = 0; off < bytes; off += 32768u)
                    bulk_g2s(dst + off, src + off, min(32768u, bytes - off), &raw_full[rs]);
            }
        } else {
            const uint32_t seg = static_cast<uint32_t>(c1 - c0) * a.cb;  // cb is a multiple of 16 here
            if (lane == 0) mbar_arrive_expect_tx(&raw_full[rs], seg * static_cast<uint32_t>(rows));
            __syncwarp();
            if (seg)
                for (int r = r0 + lane; r < r1; r += 32) {
                    const uint8_t *src =
                        a.x + ((static_cast<long long>(g.img) * a.h + (g.iy0 + r)) * a.w_ + (g.ix0 + c0)) * a.cb;
                    bulk_g2s(dst + (r - r0) * a.raw_row_bytes, src, seg, &raw_full[rs]);
                }
        }
        __syncwarp();
        ++issued;
        if (++rs == a.raw_stages) {
            rs = 0;
            ph ^= 1u;
        }
    }
    // every copy lands before the block exits
    for (int k = 0; k < a.raw_stages && k < issued; ++k) {
        if (--rs < 0) {
            rs = a.raw_stages - 1;
            ph ^= 1u;
        }
        mbar_wait_warp(&raw_full[rs], ph, a.status);
    }
}

// ---------------------------------------------------------------- converters (warps 0-3)

// Staged encoding of 8 (fp16) or 16 (e4m3) channels of one pixel.
template <int BITS>
__device__ __forceinline__ uint4 stage_cvt(const uint8_t *p)
{
    if (BITS == 8) return cvt_u8x8(*reinterpret_cast<const uint2 *>(p));
    return cvt_raw_f8<BITS>(p);
}

// Every position of the tile's window, K-chunk plane by plane: the staged
// value of the input pixel there, or the encoded zero outside the image and
// past the channel count.  Thread t owns positions t, t + 128, ... of every
// plane (their window row and column are decoded once per kernel), so a
// warp's stores are consecutive 16-byte positions.
template <int BITS>
__device__ __forceinline__ void converter_role(const WinArgs &a, uint8_t *smem, uint64_t *raw_full, uint64_t *raw_empty,
                                               uint64_t *a_full, uint64_t *a_empty)
{
    constexpr uint32_t kPad = BITS == 8 ? 0xD800D800u : 0u;  // fp16 -128.0 (x = 0), e4m3 0
    constexpr int kGroupBytes = BITS == 8 ? 8 : 16 * BITS / 8;  // packed bytes of one K-chunk
    const int tid = threadIdx.x;
    int pr[kMaxKP], pc[kMaxKP];
#pragma unroll
    for (int k = 0; k < kMaxKP; ++k) {
        const int pos = tid + 128 * k;
        pr[k] = fdiv(pos, a.fd_sp);
        pc[k] = pos - pr[k] * a.sp;
        if (pos >= a.npos) pr[k] = -1;  // no position
    }
    const int cgroups = a.c * BITS / 8 / kGroupBytes;  // K-chunks that hold input channels (c is a multiple of kch)
    int rs = 0, as = 0;
    uint32_t r_ph = 0, a_ph = 0;
    for (int t = blockIdx.x; t < a.total_tiles; t += gridDim.x) {
        const Geo g = geo_of(a, t);
        const int r0 = row_lo(a, g), r1 = row_hi(a, g);
        const int c0 = col_lo(a, g), c1 = col_hi(a, g);
        // raw column of window column px: the copied span starts at window column c0
        // (whole rows start at image column 0, i.e. window column -ix0)
        const int base_col = a.full_rows ? g.ix0 : -c0;
        uint32_t src[kMaxKP];
        bool ok[kMaxKP];
#pragma unroll
        for (int k = 0; k < kMaxKP; ++k) {
            ok[k] = pr[k] >= r0 && pr[k] < r1 && pc[k] >= c0 && pc[k] < c1;
            src[k] = ok[k] ? static_cast<uint32_t>(pr[k] - r0) * a.raw_row_bytes +
                                 static_cast<uint32_t>((pc[k] + base_col) * a.cb)
                           : 0u;
        }
        if (!mbar_wait_warp(&raw_full[rs], r_ph, a.status)) return;
        if (!mbar_wait_warp(&a_empty[as], a_ph ^ 1u, a.status)) return;
        const uint8_t *raw = smem + a.off_raw + rs * a.raw_bytes;
        const uint32_t stage = smem_addr(smem + a.off_a + as * a.stage_bytes);
        for (int gq = 0; gq < a.groups; ++gq) {
            const bool has = gq < cgroups;
            uint4 v[kMaxKP];
#pragma unroll
            for (int k = 0; k < kMaxKP; ++k) {
                // every load is issued (a safe address where the value is padding)
                const uint8_t *q = raw + ((ok[k] && has) ? src[k] + gq * kGroupBytes : 0u);
                const uint4 x = stage_cvt<BITS>(q);
                v[k] = (ok[k] && has) ? x : make_uint4(kPad, kPad, kPad, kPad);
            }
            const uint32_t plane = stage + gq * a.chunk_stride;
#pragma unroll
            for (int k = 0; k < kMaxKP; ++k)
                if (pr[k] >= 0) sts128(plane + static_cast<uint32_t>(tid + 128 * k) * 16u, v[k]);
        }
        fence_proxy_async_smem();
        mbar_arrive(&a_full[as]);
        mbar_arrive(&raw_empty[rs]);
        if (++rs == a.raw_stages) {
            rs = 0;
            r_ph ^= 1u;
        }
        if (++as == a.a_stages) {
            as = 0;
            a_ph ^= 1u;
        }
    }
}

// ---------------------------------------------------------------- MMA issue (warp 12)

template <int NT, bool F8>
__device__ __forceinline__ void mma_role(const WinArgs &a, uint8_t *smem, uint64_t *a_full, uint64_t *a_empty,
                                         uint64_t *acc_full, uint64_t *acc_empty, uint64_t *b_ready, uint64_t *done,
                                         const volatile Misc *misc)
{
    int *const status = a.status;
    bool ok = mbar_wait_warp(b_ready, 0, status);
    tc_fence_after();
    const uint32_t tmem = misc->tmem;
    const int nch = static_cast<int>(misc->nch), nslots = static_cast<int>(misc->nslots);
    const uint32_t slot_cols = misc->slot_cols;
    const uint32_t idesc = idesc_f16_f32(128, NT);  // the f16 descriptor also means e4m3 x e4m3 for kind::f8f6f4
    const uint64_t a_tmpl = smem_desc(0, a.chunk_stride, static_cast<uint32_t>(a.sp) * 16u);
    const uint64_t b_tmpl = smem_desc(0, NT * 16, 128);
    const uint32_t b16 = smem_addr(smem + a.off_b) >> 4;
    const uint32_t stages16 = smem_addr(smem + a.off_a) >> 4;
    const uint32_t kstep_a = 2u * (a.chunk_stride >> 4), kstep_b = 2u * NT;
    const uint32_t tap_b = static_cast<uint32_t>(a.groups) * NT;
    const int ct = (a.taps + nch - 1) / nch;  // taps per chunk
    const int ksteps = a.ksteps, S = a.s;
    for (int i = 0, t = blockIdx.x; ok && t < a.total_tiles; ++i, t += gridDim.x) {
        const int as = i % a.a_stages, slot = i % nslots;
        if (!mbar_wait_warp(&a_full[as], (i / a.a_stages) & 1, status)) break;
        if (!mbar_wait_warp(&acc_empty[slot], (i / nslots) & 1, status)) break;
        tc_fence_after();
        const uint32_t abase = stages16 + as * (a.stage_bytes >> 4);
        for (int s = 0; s < S; ++s) {
            for (int c = 0; c < nch; ++c) {
                const uint32_t d = tmem + slot * slot_cols + static_cast<uint32_t>(s * nch + c) * NT;
                const int t1 = min(a.taps, (c + 1) * ct);
#pragma unroll 2
                for (int tap = c * ct; tap < t1; ++tap) {
                    const uint64_t ad = a_tmpl + (abase + a.tap_a16[tap] + s * kCols);
                    const uint64_t bd = b_tmpl + (b16 + tap * tap_b);
                    for (int kk = 0; kk < ksteps; ++kk) {
                        if (F8) mma_f8_ss_warp(d, ad + kk * kstep_a, bd + kk * kstep_b, idesc, 1u);
                        else mma_f16_ss_warp(d, ad + kk * kstep_a, bd + kk * kstep_b, idesc, 1u);
                    }
                }
            }
        }
        mma_commit_warp(&acc_full[slot]);
        mma_commit_warp(&a_empty[as]);
    }
    // every issued MMA completes before TMEM is released
    mma_commit_warp(done);
    mbar_wait_warp(done, 0, status);
}

// ---------------------------------------------------------------- filter preparation (warps 4-11)

// Epilogue barrier (named barrier 1, the eight epilogue warps).
__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory"); }

// One K-chunk of one output channel's filter at one tap: the staged B row
// (8 fp16 or 16 e4m3 values in the converter's channel order) and the sums
// the compression constants and the chunk count need.
template <int BITS>
__device__ __forceinline__ uint4 filter_chunk(const uint8_t *p, bool has, int &sum, int &pos, int &neg, int &abs)
{
    if (!has) return make_uint4(0u, 0u, 0u, 0u);  // +0 in fp16 and e4m3
    if (BITS == 8) {
        const uint2 v = *reinterpret_cast<const uint2 *>(p);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int wv = static_cast<int8_t>(((k < 4 ? v.x : v.y) >> (8 * (k & 3))) & 0xFFu);
            sum += wv;
            pos += max(wv, 0);
            neg += min(wv, 0);
            abs += wv < 0 ? -wv : wv;
        }
        // byte b ^ 0x80 is the weight plus 128 as an unsigned byte: the activation encoding gives the weight
        return cvt_u8x8(make_uint2(v.x ^ 0x80808080u, v.y ^ 0x80808080u));
    }
    uint8_t e[16];
#pragma unroll
    for (int k = 0; k < 16; ++k) {
        constexpr int per = 8 / BITS;
        const int f = (p[k / per] >> ((k % per) * BITS)) & ((1 << BITS) - 1);
        const int wv = f >= (1 << (BITS - 1)) ? f - (1 << BITS) : f;
        sum += wv;
        pos += max(wv, 0);
        neg += min(wv, 0);
        abs += wv < 0 ? -wv : wv;
        // INT-2 slots follow the converter's word order (even channels, then odd, per half)
        const int slot = BITS == 4 ? k : (k & 8) + (k & 1) * 4 + ((k & 7) >> 1);
        e[slot] = e4m3_of_int(wv);
    }
    uint4 r;
    r.x = e[0] | e[1] << 8 | e[2] << 16 | static_cast<uint32_t>(e[3]) << 24;
    r.y = e[4] | e[5] << 8 | e[6] << 16 | static_cast<uint32_t>(e[7]) << 24;
    r.z = e[8] | e[9] << 8 | e[10] << 16 | static_cast<uint32_t>(e[11]) << 24;
    r.w = e[12] | e[13] << 8 | e[14] << 16 | static_cast<uint32_t>(e[15]) << 24;
    return r;
}

// The B operand ([tap][K-chunk][NT rows][16 B]), the chunk count, the
// per-channel compression records (rec0 = {lam2, kappa, shift, mode},
// rec1 = {beta, ulo, uhi, lambda}, as in the tensor-core prep kernel, with
// acc + bias = s + beta for the raw chunk sum s) and the accumulator slots.
template <int BITS, int NT>
__device__ __forceinline__ void prepare_filters(const WinArgs &a, uint8_t *smem, Misc *misc, uint64_t *b_ready)
{
    constexpr int kGroupBytes = BITS == 8 ? 8 : 16 * BITS / 8;
    constexpr int kMaxX = BITS == 8 ? 128 : (1 << BITS) - 1;  // largest |staged activation|
    const int et = threadIdx.x - kEpiWarp0 * 32;                // 0..255
    int *tapabs = reinterpret_cast<int *>(smem + a.off_tap);    // [taps][NT]
    int *sums = tapabs + a.taps * NT;                           // [3][NT]: sum, positive part, negative part
    for (int i = et; i < 3 * NT; i += kEpiWarps * 32) sums[i] = 0;
    if (et == 0) misc->mask = ~0u;
    epi_sync();
    // item i: channel n = i % NT (fixed per thread: 256 is a multiple of NT), tap i / NT
    const int cgroups = a.c * BITS / 8 / kGroupBytes;
    int sum = 0, pos = 0, neg = 0;
    const int n = et % NT;
    for (int i = et; i < a.taps * NT; i += kEpiWarps * 32) {
        const int tap = i / NT;
        int abs = 0;
        const uint8_t *src = a.w + (static_cast<long long>(n) * a.taps + tap) * (a.c * BITS / 8);
        for (int gq = 0; gq < a.groups; ++gq) {
            const uint4 v = filter_chunk<BITS>(src + gq * kGroupBytes, n < a.m && gq < cgroups, sum, pos, neg, abs);
            *reinterpret_cast<uint4 *>(smem + a.off_b + ((tap * a.groups + gq) * NT + n) * 16) = v;
        }
        tapabs[tap * NT + n] = abs;
    }
    if (a.taps * NT > et) {  // this thread saw channel n
        atomicAdd(&sums[n], sum);
        atomicAdd(&sums[NT + n], pos);
        atomicAdd(&sums[2 * NT + n], neg);
    }
    epi_sync();
    // chunk counts c = 1 .. nch_max whose even tap split keeps every chunk exact
    if (et < NT) {
        uint32_t okmask = 0;
        for (int c = 1; c <= a.nch_max; ++c) {
            const int ct = (a.taps + c - 1) / c;
            if ((c - 1) * ct >= a.taps) continue;  // an empty chunk: not a c-chunk split
            bool good = true;
            for (int j = 0; j < c && good; ++j) {
                long long b = 0;
                for (int tap = j * ct; tap < min(a.taps, (j + 1) * ct); ++tap) b += tapabs[tap * NT + et];
                good = b * kMaxX <= (1ll << 22);
            }
            if (good) okmask |= 1u << c;
        }
        okmask |= 1u << a.nch_max;  // valid for any filters by the planner's bound
        atomicAnd(&misc->mask, okmask);
    }
    epi_sync();
    const int nch = __ffs(static_cast<int>(misc->mask)) - 1;
    // per-channel records
    int4 *rec0 = reinterpret_cast<int4 *>(smem + a.off_rec);
    int4 *rec1 = rec0 + NT;
    if (et < NT) {
        const int o = et;
        const long long off = BITS == 8 ? -128 : 0;  // staged activation = x + off
        const int s_w = sums[o];
        int4 r0 = make_int4(0, 0, 0, kModeDirect), r1 = make_int4(0, 0, 0, 0);
        if (a.thr) {
            // staircase: the epilogue compares acc = s + beta with the thresholds
            const uint32_t beta = 0u - static_cast<uint32_t>(off * s_w) - static_cast<uint32_t>(nch) * kMagic;
            int32_t *ts = reinterpret_cast<int32_t *>(smem + a.off_thr) + o * kThrStride;
            for (int k = 0; k < kThrStride; ++k)
                ts[k] = (o < a.m && k < (1 << BITS) - 1) ? a.thr[static_cast<long long>(o) * ((1 << BITS) - 1) + k]
                                                        : INT32_MAX;
            r0 = make_int4(static_cast<int>(a.off_thr) + o * 4 * kThrStride, 0, 0, kModeThreshold);
            r1 = make_int4(static_cast<int32_t>(beta), 0, 0, 0);
        } else if (o < a.m) {
            const int32_t b = a.bias ? a.bias[o] : 0;
            const uint32_t beta = static_cast<uint32_t>(b) - static_cast<uint32_t>(off * s_w) -
                                  static_cast<uint32_t>(nch) * kMagic;
            const int32_t kap = a.kappa[o], lam = a.lambda[o], sh = a.shifts ? a.shifts[o] : a.shift;
            const long long top = (1 << BITS) - 1;
            // every accumulator of this channel lies in [top * neg, top * pos]
            const long long u0 = top * sums[2 * NT + o] + b, u1 = top * sums[NT + o] + b;
            const bool direct = in_i32(u0 * kap + lam) && in_i32(u1 * kap + lam);
            long long ulo = 0, uhi = 0;
            const bool clamp = !direct && saturation_bounds(kap, lam, sh, top, &ulo, &uhi);
            const int mode = direct ? kModeDirect : clamp ? kModeClamp : kModeWide;
            const uint32_t lam2 = beta * static_cast<uint32_t>(kap) + static_cast<uint32_t>(lam);
            r0 = make_int4(static_cast<int32_t>(lam2), kap, sh, mode);
            r1 = make_int4(static_cast<int32_t>(beta), static_cast<int32_t>(ulo), static_cast<int32_t>(uhi), lam);
        }
        rec0[o] = r0;
        rec1[o] = r1;
    }
    epi_sync();
    // compact direct-mode constants, and one "all direct" flag per 16-channel group
    uint2 *dcon = reinterpret_cast<uint2 *>(rec1 + NT);
    uint8_t *gd = reinterpret_cast<uint8_t *>(dcon + NT);
    if (et < NT) {
        const int4 r0 = rec0[et];
        dcon[et] = make_uint2(static_cast<uint32_t>(r0.x),
                              (static_cast<uint32_t>(r0.y) & 0xFFFFu) | (static_cast<uint32_t>(r0.z) << 16));
    }
    if (et < NT / 16) {
        int all = 1;
        for (int k = 0; k < 16; ++k) all &= rec0[et * 16 + k].w == kModeDirect;
        gd[et] = static_cast<uint8_t>(all);
    }
    // B was written through the generic proxy; the tensor cores read it through the async proxy
    fence_proxy_async_smem();
    epi_sync();
    if (et == 0) {
        const uint32_t cols = static_cast<uint32_t>(a.s * nch * NT);
        misc->nch = static_cast<uint32_t>(nch);
        misc->slot_cols = cols;
        misc->nslots = min(static_cast<uint32_t>(kMaxSlots), 512u / cols);
        mbar_arrive(b_ready);
    }
    epi_sync();
}

// ---------------------------------------------------------------- epilogue (warps 4-11)

template <int CW>
__device__ __forceinline__ void tmem_fill(uint32_t taddr)
{
    if (CW == 8) {
        tmem_st8_fill(taddr, kMagic);
    } else {
#pragma unroll
        for (int c = 0; c < CW; c += 16) tmem_st16_fill(taddr + c, kMagic);
    }
}

// The integer sum of the chunks' bit patterns of EB consecutive columns of one
// strip (chunk buffers `stride` columns apart), each buffer's columns refilled
// with the pre-load once read.  NCH > 0: that many chunks, each chunk's loads
// in flight before one wait; NCH = 0: any count.
template <int EB, int NCH>
__device__ __forceinline__ void drain(uint32_t addr, uint32_t stride, int nch, uint32_t (&v)[EB])
{
    constexpr int L = EB < 16 ? 8 : 16;  // columns per TMEM load
    const int n = NCH > 0 ? NCH : nch;
#pragma unroll(NCH > 0 ? NCH : 1)
    for (int c = 0; c < n; ++c) {
        uint32_t t[EB];
#pragma unroll
        for (int b0 = 0; b0 < EB; b0 += L) {
            if constexpr (L == 16) tmem_ld16(addr + c * stride + b0, *reinterpret_cast<uint32_t(*)[16]>(t + b0));
            else tmem_ld8(addr + c * stride + b0, *reinterpret_cast<uint32_t(*)[8]>(t + b0));
        }
        tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < EB; ++k) v[k] = c == 0 ? t[k] : v[k] + t[k];
        tmem_fill<EB>(addr + c * stride);
    }
}

// Compression (Sec. III-A) of G raw chunk sums of one pixel and Q-bit packing.
// Direct channels use the compact constants dcon = {lam2, kappa | shift << 16}:
// ((s * kappa + lam2) mod 2^32) >> shift is exact there (see the records).
template <int BITS, int G>
__device__ __forceinline__ void win_compress(const uint32_t *s, const uint2 *dcon, const int4 *rec0, const int4 *rec1,
                                             bool direct, int m_first, uint32_t (&packed)[(G * BITS + 31) / 32])
{
    int y[G];
    if (direct) {
#pragma unroll
        for (int k = 0; k < G; ++k) {
            const uint2 d = dcon[m_first + k];
            const uint32_t kap = static_cast<uint32_t>(static_cast<int32_t>(static_cast<int16_t>(d.y & 0xFFFFu)));
            y[k] = static_cast<int32_t>(s[k] * kap + d.x) >> (d.y >> 16);
        }
    } else {
#pragma unroll
        for (int k = 0; k < G; ++k)
            y[k] = static_cast<int>(compress_slow(s[k], rec0[m_first + k], rec1[m_first + k], (1u << BITS) - 1u));
    }
    constexpr int kPer = 32 / BITS;
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

template <int BITS, int NT, bool POOL>
__device__ __forceinline__ void epilogue_role(const WinArgs &a, uint8_t *smem, uint64_t *acc_full, uint64_t *acc_empty,
                                              const Misc *misc)
{
    constexpr int CW = NT / 2;           // columns of this warp
    constexpr int EB = CW < 32 ? CW : 32;  // columns drained and compressed together
    constexpr int G = EB < 16 ? EB : 16;   // channels per compression group
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quarter = warp & 3, half = (warp - kEpiWarp0) >> 2;
    const int row = quarter * 32 + lane;  // tile row of the strip: 8 * (output row) + column
    const int col0 = half * CW;
    const uint32_t tmem = misc->tmem;
    const int nch = static_cast<int>(misc->nch), nslots = static_cast<int>(misc->nslots);
    const uint32_t slot_cols = misc->slot_cols;
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + col0;
    const int4 *rec0 = reinterpret_cast<const int4 *>(smem + a.off_rec);
    const int4 *rec1 = rec0 + NT;
    const uint2 *dcon = reinterpret_cast<const uint2 *>(rec1 + NT);
    const uint8_t *gdirect = reinterpret_cast<const uint8_t *>(dcon + NT);
    const int out_row_bytes = a.m * BITS / 8;
    const int S = a.s;
    int *const status = a.status;

    // every buffer this warp reads starts at the pre-load; then all slots are free
    for (int slot = 0; slot < nslots; ++slot)
        for (int b = 0; b < S * nch; ++b) tmem_fill<CW>(lane_addr + slot * slot_cols + b * NT);
    tmem_wait_st();
    tc_fence_before();
    __syncwarp();
    if (lane == 0)
        for (int slot = 0; slot < nslots; ++slot) mbar_arrive(&acc_empty[slot]);

    const int oyr = row >> 3, oxr = row & 7;
    for (int i = 0, t = blockIdx.x; t < a.total_tiles; ++i, t += gridDim.x) {
        const int slot = i % nslots;
        const Geo g = geo_of(a, t);
        if (!mbar_wait_warp(&acc_full[slot], (i / nslots) & 1, status)) return;
        tc_fence_after();
        const int oy = g.oy0 + oyr;
        for (int s = 0; s < S; ++s) {
            const int ox = g.ox0 + s * kCols + oxr;
            const bool pix_ok = oy < a.oh && ox < a.ow;
            // Fused 2x2/2 max-pool: pooled pixel (oy/2, ox/2) is the window of lanes
            // L, L^1, L^8, L^9; its top-left lane stores.
            const bool pool_store = POOL && (row & 9) == 0 && (oy >> 1) < a.pool_oh && (ox >> 1) < a.pool_ow;
            uint8_t *dst = POOL ? a.y + ((static_cast<long long>(g.img) * a.pool_oh + (oy >> 1)) * a.pool_ow + (ox >> 1)) *
                                            out_row_bytes
                                : a.y + ((static_cast<long long>(g.img) * a.oh + oy) * a.ow + ox) * out_row_bytes;
#pragma unroll
            for (int k0 = 0; k0 < CW; k0 += EB) {
                uint32_t v[EB];
                const uint32_t src = lane_addr + slot * slot_cols + static_cast<uint32_t>(s * nch) * NT + k0;
                if (nch == 1) drain<EB, 1>(src, NT, 1, v);
                else if (nch == 2) drain<EB, 2>(src, NT, 2, v);
                else drain<EB, 0>(src, NT, nch, v);
                if (s == S - 1 && k0 + EB == CW) {  // the slot's last columns are read: give it back first
                    tmem_wait_st();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&acc_empty[slot]);
                }
#pragma unroll
                for (int c = 0; c < EB; c += G) {
                    const int m0 = col0 + k0 + c;
                    const int valid = a.m - m0;  // same for the whole warp
                    if (valid <= 0) continue;
                    uint32_t pk[(G * BITS + 31) / 32];
                    win_compress<BITS, G>(v + c, dcon, rec0, rec1, gdirect[m0 >> 4] != 0, m0, pk);
                    if constexpr (POOL) {
#pragma unroll
                        for (int wd = 0; wd < (G * BITS + 31) / 32; ++wd) {  // every lane shuffles
                            pk[wd] = max_fields<BITS>(pk[wd], __shfl_xor_sync(0xffffffffu, pk[wd], 1));
                            pk[wd] = max_fields<BITS>(pk[wd], __shfl_xor_sync(0xffffffffu, pk[wd], 8));
                        }
                        if (pool_store) store_packed<BITS, G>(pk, valid, dst + m0 * BITS / 8);
                    } else if (pix_ok) {
                        store_packed<BITS, G>(pk, valid, dst + m0 * BITS / 8);
                    }
                }
            }
        }
    }
}

// ---------------------------------------------------------------- the kernel

template <int BITS, int NT, bool POOL>
__global__ void __launch_bounds__(kThreads, 1) conv_win_kernel(const WinArgs a)
{
    extern __shared__ __align__(128) uint8_t smem[];
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + a.off_bar);
    uint64_t *raw_full = bars;
    uint64_t *raw_empty = raw_full + kMaxStages;
    uint64_t *a_full = raw_empty + kMaxStages;
    uint64_t *a_empty = a_full + kMaxStages;
    uint64_t *acc_full = a_empty + kMaxStages;
    uint64_t *acc_empty = acc_full + kMaxSlots;
    uint64_t *b_ready = acc_empty + kMaxSlots;
    uint64_t *done = b_ready + 1;
    Misc *misc = reinterpret_cast<Misc *>(done + 1);
    const int warp = threadIdx.x >> 5;

    if (warp == kMmaWarp) {
        if ((threadIdx.x & 31) == 0) {
            for (int s = 0; s < kMaxStages; ++s) {
                mbar_init(&raw_full[s], 1);
                mbar_init(&raw_empty[s], kConvWarps * 32);
                mbar_init(&a_full[s], kConvWarps * 32);
                mbar_init(&a_empty[s], 1);
            }
            for (int b = 0; b < kMaxSlots; ++b) {
                mbar_init(&acc_full[b], 1);
                mbar_init(&acc_empty[b], kEpiWarps);
            }
            mbar_init(b_ready, 1);
            mbar_init(done, 1);
            fence_mbar_init();
        }
        __syncwarp();
        tmem_alloc(&misc->tmem, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    if (warp < kConvWarps) {
        converter_role<BITS>(a, smem, raw_full, raw_empty, a_full, a_empty);
    } else if (warp < kConvWarps + kEpiWarps) {
        prepare_filters<BITS, NT>(a, smem, misc, b_ready);
        epilogue_role<BITS, NT, POOL>(a, smem, acc_full, acc_empty, misc);
    } else if (warp == kMmaWarp) {
        mma_role<NT, BITS != 8>(a, smem, a_full, a_empty, acc_full, acc_empty, b_ready, done, misc);
    } else if (warp == kLoadWarp) {
        loader_role(a, smem, raw_full, raw_empty);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(misc->tmem, 512);
    }
}

}  // namespace win

// Launch of one instantiation (defined per bit width in conv_win_q*.cu).
template <int BITS>
cudaError_t launch_win_bits(const win::WinArgs &a, int nt, int grid, uint32_t smem, cudaStream_t st);

}  // namespace qnn
