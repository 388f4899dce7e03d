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
// With few input channels (INT-8, c * kw <= 16) the kernel columns fold into
// K instead: a staged position holds the c channels of kw neighbouring pixels,
// the window is 8S positions wide and each MMA covers one kernel row.
//
// Exactness on fp16 / e4m3 tensor cores (there is no integer tcgen05 MMA on
// this GPU).  INT-8 activations are staged as x - 128 in fp16, INT-4 / INT-2
// as themselves in e4m3; weights as themselves; all exact.  Every accumulator
// starts at 1.5 * 2^23, written by one fp16 MMA that overwrites it with
// 2048 * 6144 (both exact in fp16, their product exact in fp32) ahead of the
// layer's MMAs, so no TMEM store is needed; while the partial sums of a chunk stay
// within 2^22 of it every one is an integer that fp32 holds exactly; the bit
// pattern minus the pre-load is the chunk's integer sum.  The kernel derives
// the number of chunks from the filters themselves: the fewest contiguous tap
// ranges for which max|staged x| * sum|w| over the range stays within 2^22 for
// every output channel (the worst case over all filters is the planner's
// nch_max, always valid).
//
// Filters in the kernel.  The loader first bulk-copies the packed filters and
// the first windows' input rows; meanwhile the epilogue warps and the MMA warp
// turn the filters into the B operand (K-major core matrices) and derive the
// chunk count and the MMA issue order, and the epilogue warps the per-channel
// compression records, all in shared memory, while the converters stage the
// first windows.  So one qconv_hwc call is one launch and needs no workspace.
// qconv_hwc_prepare runs the same preparation once, in a one-block launch
// that writes the resulting shared-memory image to a workspace, and each
// qconv_hwc_run launch copies that image instead of preparing.
//
// Warp roles after that (one persistent CTA per SM, 14 warps):
//   warps 0-3   converters: raw window -> staged operand, every position
//   warps 4-11  epilogue: warp w reads TMEM lane quarter w % 4 and one half
//               of the output channels; sums the chunks, compresses, packs at
//               Q bits and stores
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
// the filter preparation runs on the epilogue warps and the MMA warp (the
// warps that use its results), synchronised by named barrier 1; the
// converters and the loader start on the first windows meanwhile
constexpr int kPrepWarp0 = kEpiWarp0;
constexpr int kPrepThreads = (kMmaWarp + 1 - kPrepWarp0) * 32;
constexpr int kRows = 16, kCols = 8;  // output rows and columns of one strip
constexpr int kMaxTaps = 64;
constexpr int kMaxSlots = 4;          // accumulator slots in TMEM
constexpr int kMaxStages = 4;         // raw windows / staged windows in flight
constexpr int kMaxKP = 5;             // window positions per converter thread and K-chunk plane
constexpr int kSmemLimit = 232448;    // 227 KB opt-in dynamic shared memory per block

// Shared-memory words after the barriers: the TMEM base, the chunk count the
// filters allow, the accumulator slot count and width, the chunk-mask vote,
// the MMAs per tile.
struct Misc {
    uint32_t tmem;
    uint32_t nch;  // accumulators per strip: exact chunks x K-split
    uint32_t nslots;
    uint32_t slot_cols;
    uint32_t mask;
    uint32_t nmma;  // MMAs per tile (entries of the issue table)
    uint32_t kx;    // K-split: the k-steps of a tap alternate between kx accumulators
    uint32_t cst;   // TMEM column of the per-channel constants (lam2, then kappa), or ~0u: none
};

// Accumulator slots of `cols` columns each, and the 2 * NT columns of the
// per-channel constants behind them when two slots still fit.
template <int NT>
__device__ __forceinline__ void slot_layout(Misc *misc, uint32_t cols)
{
    uint32_t ns = min(static_cast<uint32_t>(kMaxSlots), (512u - 2u * NT) / cols);
    uint32_t cst = ns * cols;
    if (ns < 2) {
        ns = min(static_cast<uint32_t>(kMaxSlots), 512u / cols);
        cst = ~0u;
    }
    misc->slot_cols = cols;
    misc->nslots = ns;
    misc->cst = cst;
}

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
    int fold;                // kernel columns folded into K: a tap is a kernel row (INT-8, c * kw <= 16)
    int kwf;                 // kernel columns as the MMAs see them (1 when folded)
    int cb;                  // packed bytes per input pixel
    int full_rows;
    int tiles_x, tiles_per_img, total_tiles;
    FastDiv fd_tpi, fd_tx, fd_sp;
    int raw_stages, a_stages, nch_max, nch_min;
    uint32_t raw_row_bytes, raw_bytes, chunk_stride, stage_bytes;
    uint32_t off_b, off_a, off_raw, off_rec, off_thr, off_tap, off_bar;
    uint32_t off_wraw, wraw_bytes;  // packed filters copied into shared memory (0 bytes: read from global)
    uint32_t off_mtab;              // the MMA issue table (S * taps * ksteps entries of 8 bytes)
    uint32_t off_pre;               // operands of the pre-load MMA (A 4 KB, then B 2 * NT * 16 bytes)
    // The prepared image: B ([off_b, off_b + b_bytes)) followed by the tail
    // [off_rec, off_rec + tail_bytes) (records, thresholds, tap sums with the
    // chunk count, MMA table, pre-load operands).  img: read it instead of
    // preparing the filters; img_out: prepare, write it and stop (one block).
    const uint8_t *img;
    uint8_t *img_out;
    uint32_t b_bytes, tail_bytes;
    int pool, pool_oh, pool_ow;
    int *status;
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

// The loader's position in its ring of raw windows.
struct LoadState {
    int rs, issued, t;
    uint32_t ph;
};

// The packed filters, copied into shared memory for the filter preparation.
__device__ __forceinline__ void load_filters(const WinArgs &a, uint8_t *smem, uint64_t *w_full)
{
    if (a.wraw_bytes && (threadIdx.x & 31) == 0) {
        mbar_arrive_expect_tx(w_full, a.wraw_bytes);
        for (uint32_t off = 0; off < a.wraw_bytes; off += 32768u)
            bulk_g2s(smem + a.off_wraw + off, a.w + off, min(32768u, a.wraw_bytes - off), w_full);
    }
    __syncwarp();
}

// The input rows of up to `count` more tiles' windows: one bulk copy when
// windows span whole image rows, else one per row (lanes issue them in
// parallel).
__device__ __forceinline__ void load_windows(const WinArgs &a, uint8_t *smem, uint64_t *raw_full, uint64_t *raw_empty,
                                             LoadState &st, int count)
{
    const int lane = threadIdx.x & 31;
    for (; st.t < a.total_tiles && count > 0; st.t += gridDim.x, --count) {
        const Geo g = geo_of(a, st.t);
        const int r0 = row_lo(a, g), r1 = row_hi(a, g);
        const int c0 = col_lo(a, g), c1 = col_hi(a, g);
        if (!mbar_wait_warp(&raw_empty[st.rs], st.ph ^ 1u, a.status)) {
            st.t = a.total_tiles;  // give up: the other roles time out as well
            break;
        }
        uint8_t *dst = smem + a.off_raw + st.rs * a.raw_bytes;
        const int rows = r1 - r0;
        if (a.full_rows) {
            const uint32_t bytes = static_cast<uint32_t>(rows) * a.raw_row_bytes;
            if (lane == 0) {
                mbar_arrive_expect_tx(&raw_full[st.rs], bytes);
                const uint8_t *src = a.x + (static_cast<long long>(g.img) * a.h + (g.iy0 + r0)) * a.raw_row_bytes;
                for (uint32_t off = 0; off < bytes; off += 32768u)
                    bulk_g2s(dst + off, src + off, min(32768u, bytes - off), &raw_full[st.rs]);
            }
        } else {
            const uint32_t seg = static_cast<uint32_t>(c1 - c0) * a.cb;  // cb is a multiple of 16 here
            if (lane == 0) mbar_arrive_expect_tx(&raw_full[st.rs], seg * static_cast<uint32_t>(rows));
            __syncwarp();
            if (seg)
                for (int r = r0 + lane; r < r1; r += 32) {
                    const uint8_t *src =
                        a.x + ((static_cast<long long>(g.img) * a.h + (g.iy0 + r)) * a.w_ + (g.ix0 + c0)) * a.cb;
                    bulk_g2s(dst + (r - r0) * a.raw_row_bytes, src, seg, &raw_full[st.rs]);
                }
        }
        __syncwarp();
        ++st.issued;
        if (++st.rs == a.raw_stages) {
            st.rs = 0;
            st.ph ^= 1u;
        }
    }
}

// Every copy lands before the block exits.
__device__ __forceinline__ void load_drain(const WinArgs &a, uint64_t *raw_full, uint64_t *w_full, LoadState st)
{
    for (int k = 0; k < a.raw_stages && k < st.issued; ++k) {
        if (--st.rs < 0) {
            st.rs = a.raw_stages - 1;
            st.ph ^= 1u;
        }
        mbar_wait_warp(&raw_full[st.rs], st.ph, a.status);
    }
    if (a.wraw_bytes) mbar_wait_warp(w_full, 0, a.status);
}

// ---------------------------------------------------------------- converters (warps 0-3)

// Staged encoding of one K-chunk of a pixel from its packed bytes: 8 unsigned
// bytes -> 8 fp16 (x - 128), or 16 nibbles / crumbs -> 16 e4m3 (the channel
// orders of cvt_raw_f8, which the filter layout follows).
template <int BITS>
__device__ __forceinline__ uint4 stage_chunk(uint2 v)
{
    if (BITS == 8) return cvt_u8x8(v);
    if (BITS == 4) return make_uint4(e4m3x4(v.x), e4m3x4(v.x >> 16), e4m3x4(v.y), e4m3x4(v.y >> 16));
    const uint32_t ev = v.x & 0x33333333u, od = (v.x >> 2) & 0x33333333u;  // crumbs 2k and 2k+1 as nibbles
    return make_uint4(e4m3x4(ev), e4m3x4(od), e4m3x4(ev >> 16), e4m3x4(od >> 16));
}

// Every position of the tile's window: the staged value of the input pixel
// there, or the encoded zero outside the image and past the channel count.
// Thread t owns positions t, t + 128, ...; per position it loads the pixel's
// packed channels (16-byte loads when a pixel is a whole number of 16-byte
// units, else 8-byte ones) and stores one 16-byte chunk per K-chunk plane, so
// a warp's stores are consecutive positions of a plane.
template <int BITS>
__device__ __forceinline__ void converter_role(const WinArgs &a, uint8_t *smem, uint64_t *raw_full, uint64_t *raw_empty,
                                               uint64_t *a_full, uint64_t *a_empty)
{
    constexpr uint32_t kPad = BITS == 8 ? 0xD800D800u : 0u;  // fp16 -128.0 (x = 0), e4m3 0
    constexpr int kGroupBytes = BITS == 8 ? 8 : 16 * BITS / 8;  // packed bytes of one K-chunk
    const int tid = threadIdx.x;
    const int cgroups = a.c * BITS / 8 / kGroupBytes;  // K-chunks that hold input channels (c is a multiple of kch)
    const int groups = a.groups;
    const int words = a.cb / 8;             // 8-byte words of one pixel (at most 8)
    const bool wide = (a.cb & 15) == 0;     // 16-byte aligned pixels
    int rs = 0, as = 0;
    uint32_t r_ph = 0, a_ph = 0;
    for (int t = blockIdx.x; t < a.total_tiles; t += gridDim.x) {
        const Geo g = geo_of(a, t);
        const int r0 = row_lo(a, g), r1 = row_hi(a, g);
        const int c0 = col_lo(a, g), c1 = col_hi(a, g);
        // raw column of window column px: the copied span starts at window column c0
        // (whole rows start at image column 0, i.e. window column -ix0)
        const int base_col = a.full_rows ? g.ix0 : -c0;
        if (!mbar_wait_warp(&raw_full[rs], r_ph, a.status)) return;
        if (!mbar_wait_warp(&a_empty[as], a_ph ^ 1u, a.status)) return;
        const uint8_t *raw = smem + a.off_raw + rs * a.raw_bytes;
        const uint32_t stage = smem_addr(smem + a.off_a + as * a.stage_bytes);
        // Three positions per iteration, every load of the three issued before any
        // conversion (shared memory is busy with the tensor cores' operand reads,
        // so each round trip is long); one loop body keeps the code of the four
        // roles running side by side on each SM sub-partition small.
#pragma unroll 1
        for (int pos0 = tid; pos0 < a.npos; pos0 += 3 * 128) {
            uint2 pv[3][8];
            bool ok[3];
#pragma unroll
            for (int u = 0; u < 3; ++u) {
                const int pos = pos0 + u * 128;
                const int pr = fdiv(pos, a.fd_sp), pc = pos - pr * a.sp;
                ok[u] = pos < a.npos && pr >= r0 && pr < r1 && pc >= c0 && pc < c1;
                // the pixel's packed channels (a safe address where the value is padding)
                const uint8_t *q = raw + (ok[u] ? static_cast<uint32_t>(pr - r0) * a.raw_row_bytes +
                                                      static_cast<uint32_t>((pc + base_col) * a.cb)
                                                : 0u);
                if (wide) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const uint4 v = 2 * j < words ? *reinterpret_cast<const uint4 *>(q + 16 * j) : make_uint4(0, 0, 0, 0);
                        pv[u][2 * j] = make_uint2(v.x, v.y);
                        pv[u][2 * j + 1] = make_uint2(v.z, v.w);
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        pv[u][j] = j < words ? *reinterpret_cast<const uint2 *>(q + 8 * j) : make_uint2(0, 0);
                }
            }
#pragma unroll
            for (int u = 0; u < 3; ++u) {
                const int pos = pos0 + u * 128;
                if (pos >= a.npos) break;
                const uint32_t pos16 = static_cast<uint32_t>(pos) * 16u;
#pragma unroll
                for (int gq = 0; gq < 8; ++gq) {
                    if (gq >= groups) break;
                    uint2 v;
                    if (kGroupBytes == 8) v = pv[u][gq];
                    else v = make_uint2((gq & 1) ? pv[u][gq >> 1].y : pv[u][gq >> 1].x, 0u);
                    const uint4 x = stage_chunk<BITS>(v);
                    const bool real = ok[u] && gq < cgroups;
                    sts128(stage + gq * a.chunk_stride + pos16, real ? x : make_uint4(kPad, kPad, kPad, kPad));
                }
            }
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

// The folded layout (INT-8, kernel columns folded into K): position (row, col)
// of the window holds the kw * c bytes of image pixels col .. col + kw - 1 of
// its row, then zeros, staged as 16 fp16 values x - 128 in two K-chunk planes;
// kernel row i of strip s reads the window i rows and 8s positions on.  The
// raw stage holds whole image rows.  Activation 0 stands outside the image
// (it stages as -128, like every padded value); the values past kw * c meet
// zero weights.
__device__ __forceinline__ void converter_fold(const WinArgs &a, uint8_t *smem, uint64_t *raw_full,
                                               uint64_t *raw_empty, uint64_t *a_full, uint64_t *a_empty)
{
    const int tid = threadIdx.x;
    int rs = 0, as = 0;
    uint32_t r_ph = 0, a_ph = 0;
    for (int t = blockIdx.x; t < a.total_tiles; t += gridDim.x) {
        const Geo g = geo_of(a, t);
        const int r0 = row_lo(a, g), r1 = row_hi(a, g);
        if (!mbar_wait_warp(&raw_full[rs], r_ph, a.status)) return;
        if (!mbar_wait_warp(&a_empty[as], a_ph ^ 1u, a.status)) return;
        const uint8_t *raw = smem + a.off_raw + rs * a.raw_bytes;
        const uint32_t stage = smem_addr(smem + a.off_a + as * a.stage_bytes);
#pragma unroll 1
        for (int pos = tid; pos < a.npos; pos += 128) {
            const int pr = fdiv(pos, a.fd_sp), pc = pos - pr * a.sp;
            const int col = g.ix0 + pc;  // image column of the position's first pixel
            // the span's pixels inside the image, [jlo, jhi); their bytes are contiguous in the row
            const int jlo = max(0, -col), jhi = min(a.kw, a.w_ - col);
            unsigned long long lo = 0ull, hi = 0ull;  // the 16 bytes, zero outside the image
            if (pr >= r0 && pr < r1 && jhi > jlo) {
                const uint8_t *row = raw + static_cast<uint32_t>(pr - r0) * a.raw_row_bytes;
                // five aligned words from the first inside byte, funnel-shifted to it
                const uint32_t off = static_cast<uint32_t>((col + jlo) * a.c);
                const uint32_t *wp = reinterpret_cast<const uint32_t *>(row + (off & ~3u));
                uint32_t q[5];
#pragma unroll
                for (int k = 0; k < 5; ++k) q[k] = wp[k];
                const uint32_t sh = (off & 3u) * 8u;
                lo = static_cast<unsigned long long>(__funnelshift_r(q[0], q[1], sh)) |
                     static_cast<unsigned long long>(__funnelshift_r(q[1], q[2], sh)) << 32;
                hi = static_cast<unsigned long long>(__funnelshift_r(q[2], q[3], sh)) |
                     static_cast<unsigned long long>(__funnelshift_r(q[3], q[4], sh)) << 32;
                // to byte jlo * c of the span (a 128-bit shift), then keep bytes [jlo * c, jhi * c)
                const int s8 = jlo * a.c * 8;
                if (s8 >= 64) {
                    hi = lo << (s8 - 64);
                    lo = 0ull;
                } else if (s8 > 0) {
                    hi = (hi << s8) | (lo >> (64 - s8));
                    lo <<= s8;
                }
                const int b1 = jhi * a.c;  // bytes below b1 stay
                const unsigned long long keep_lo = b1 >= 8 ? ~0ull : (1ull << (8 * b1)) - 1ull;
                const unsigned long long keep_hi = b1 >= 16 ? ~0ull : b1 <= 8 ? 0ull : (1ull << (8 * (b1 - 8))) - 1ull;
                lo &= keep_lo;
                hi &= keep_hi;
            }
            uint32_t wd[4] = {static_cast<uint32_t>(lo), static_cast<uint32_t>(lo >> 32), static_cast<uint32_t>(hi),
                              static_cast<uint32_t>(hi >> 32)};
            const uint32_t pos16 = static_cast<uint32_t>(pos) * 16u;
            sts128(stage + pos16, cvt_u8x8(make_uint2(wd[0], wd[1])));
            sts128(stage + a.chunk_stride + pos16, cvt_u8x8(make_uint2(wd[2], wd[3])));
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

__device__ __forceinline__ uint64_t desc_of(uint32_t lo, uint32_t hi)
{
    return (static_cast<uint64_t>(hi) << 32) | lo;
}

template <bool F8>
__device__ __forceinline__ void mma_nc(uint32_t d, uint64_t ad, uint64_t bd, uint32_t idesc)
{
    if (F8) mma_f8_ss_warp_nc(d, ad, bd, idesc, 1u);
    else mma_f16_ss_warp_nc(d, ad, bd, idesc, 1u);
}

// One tile's MMAs with every offset known at compile time (one exact chunk,
// KH x KW taps, KS k-steps per tap, S strips, k-step kk of a tap into the
// strip's accumulator kk % KX): a descriptor is its template's low word plus
// an offset (a start address field that cannot carry out of its 14 bits), so
// each MMA costs an addition or two and the issue.  Consecutive MMAs go to
// S * KX different accumulators: an MMA into the accumulator the previous one
// wrote waits for it, so one chain runs at about half the tensor pipe's rate.
template <int KH, int KW, int KS, int S, int NT, bool F8, int KX>
__device__ __forceinline__ void issue_fixed(uint32_t d0, uint32_t alo, uint32_t ahi, uint32_t blo, uint32_t bhi,
                                            uint32_t idesc, int sp, uint32_t kstep_a)
{
    // one kernel row per iteration: its KW * KS * S MMAs unrolled
#pragma unroll 1
    for (int i = 0; i < KH; ++i) {
        const uint32_t arow = alo + static_cast<uint32_t>(i * sp);
#pragma unroll
        for (int j = 0; j < KW; ++j)
#pragma unroll
            for (int kk = 0; kk < KS; ++kk) {
                const uint64_t bd = desc_of(blo + static_cast<uint32_t>(((i * KW + j) * 2 * KS + 2 * kk) * NT), bhi);
#pragma unroll
                for (int s = 0; s < S; ++s)
                    mma_nc<F8>(d0 + (s * KX + kk % KX) * NT, desc_of(arow + j + kk * kstep_a + s * kCols, ahi), bd,
                               idesc);
            }
    }
}

template <int NT, bool F8>
__device__ __forceinline__ void mma_role(const WinArgs &a, uint8_t *smem, uint64_t *a_full, uint64_t *a_empty,
                                         uint64_t *acc_full, uint64_t *acc_empty, uint64_t *done, const Misc *misc)
{
    int *const status = a.status;
    const uint32_t tmem = misc->tmem;
    const int nch = static_cast<int>(misc->nch), nslots = static_cast<int>(misc->nslots);
    const uint32_t slot_cols = misc->slot_cols;
    const uint32_t idesc = idesc_f16_f32(128, NT);  // the f16 descriptor also means e4m3 x e4m3 for kind::f8f6f4
    const uint64_t a_tmpl = smem_desc(0, a.chunk_stride, static_cast<uint32_t>(a.sp) * 16u);
    const uint64_t b_tmpl = smem_desc(0, NT * 16, 128);
    const uint32_t b16 = smem_addr(smem + a.off_b) >> 4;
    const uint32_t stages16 = smem_addr(smem + a.off_a) >> 4;
    const uint32_t kstep_a = 2u * (a.chunk_stride >> 4);
    // the pre-load MMA: fp16 operands in shared memory, accumulate = 0
    const uint32_t pre16 = smem_addr(smem + a.off_pre) >> 4;
    const uint64_t pre_a = smem_desc(0, 2048, 128) + pre16;
    const uint64_t pre_b = smem_desc(0, NT * 16, 128) + pre16 + 256;
    const int nacc = a.s * nch;
    const int kx = static_cast<int>(misc->kx);
    // the issue order (built by the filter preparation): one 8-byte entry per MMA,
    // {A offset in 16-byte units | accumulator column << 16, B offset}
    const uint2 *tab = reinterpret_cast<const uint2 *>(smem + a.off_mtab);
    const int nu = static_cast<int>(misc->nmma);
    // the common shapes with one exact chunk issue from unrolled code
    const int fixed = nch != kx ? 0
                      : (a.kh == 3 && a.kwf == 3 && a.ksteps == 2 && a.s == 2) ? 1
                      : (a.kh == 3 && a.kwf == 3 && a.ksteps == 1 && a.s == 2) ? 2
                      : (a.kh == 5 && a.kwf == 5 && a.ksteps == 2 && a.s == 2) ? 3
                      : (a.kh == 5 && a.kwf == 5 && a.ksteps == 2 && a.s == 1) ? 4
                      : (a.kh == 3 && a.kwf == 3 && a.ksteps == 4 && a.s == 2) ? 5
                                                                                : 0;
    for (int i = 0, t = blockIdx.x; t < a.total_tiles; ++i, t += gridDim.x) {
        const int as = i % a.a_stages, slot = i % nslots;
        if (!mbar_wait_warp(&a_full[as], (i / a.a_stages) & 1, status)) break;
        if (!mbar_wait_warp(&acc_empty[slot], (i / nslots) & 1, status)) break;
        tc_fence_after();
        const uint64_t abase = a_tmpl + (stages16 + as * (a.stage_bytes >> 4));
        const uint64_t bbase = b_tmpl + b16;
        const uint32_t d0 = tmem + slot * slot_cols;
        // every accumulator of the slot starts at the pre-load (accumulate = 0)
        for (int b = 0; b < nacc; ++b) mma_f16_ss_warp_nc(d0 + b * NT, pre_a, pre_b, idesc, 0u);
        const uint32_t alo = static_cast<uint32_t>(abase), ahi = static_cast<uint32_t>(abase >> 32);
        const uint32_t blo = static_cast<uint32_t>(bbase), bhi = static_cast<uint32_t>(bbase >> 32);
        switch (fixed * 2 + (kx == 2 ? 1 : 0)) {
            case 2: issue_fixed<3, 3, 2, 2, NT, F8, 1>(d0, alo, ahi, blo, bhi, idesc, a.sp, kstep_a); break;
            case 3: issue_fixed<3, 3, 2, 2, NT, F8, 2>(d0, alo, ahi, blo, bhi, idesc, a.sp, kstep_a); break;
            case 4: issue_fixed<3, 3, 1, 2, NT, F8, 1>(d0, alo, ahi, blo, bhi, idesc, a.sp, kstep_a); break;
            case 6: issue_fixed<5, 5, 2, 2, NT, F8, 1>(d0, alo, ahi, blo, bhi, idesc, a.sp, kstep_a); break;
            case 7: issue_fixed<5, 5, 2, 2, NT, F8, 2>(d0, alo, ahi, blo, bhi, idesc, a.sp, kstep_a); break;
            case 8: issue_fixed<5, 5, 2, 1, NT, F8, 1>(d0, alo, ahi, blo, bhi, idesc, a.sp, kstep_a); break;
            case 9: issue_fixed<5, 5, 2, 1, NT, F8, 2>(d0, alo, ahi, blo, bhi, idesc, a.sp, kstep_a); break;
            case 10: issue_fixed<3, 3, 4, 2, NT, F8, 1>(d0, alo, ahi, blo, bhi, idesc, a.sp, kstep_a); break;
            case 11: issue_fixed<3, 3, 4, 2, NT, F8, 2>(d0, alo, ahi, blo, bhi, idesc, a.sp, kstep_a); break;
            default:
#pragma unroll 4
                for (int u = 0; u < nu; ++u) {
                    const uint2 e = tab[u];
                    mma_nc<F8>(d0 + (e.x >> 16), abase + (e.x & 0xFFFFu), bbase + e.y, idesc);
                }
        }
        mma_commit_warp(&acc_full[slot]);
        mma_commit_warp(&a_empty[as]);
    }
    // every issued MMA completes before TMEM is released
    mma_commit_warp(done);
    mbar_wait_warp(done, 0, status);
}

// ---------------------------------------------------------------- filter preparation (warps 4-12)

__device__ __forceinline__ void prep_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kPrepThreads) : "memory"); }

// One K-chunk of one output channel's filter at one tap, from its packed
// bytes (8, or 4 at INT-2, in v): the staged B row (8 fp16 or 16 e4m3 values
// in the converter's channel order) and the sums the compression constants and
// the chunk count need.
template <int BITS>
__device__ __forceinline__ uint4 filter_chunk(uint2 v, int &pos, int &neg, int &abs)
{
    if constexpr (BITS == 8) {
        // byte sums by 4-way signed dot products with ones: all weights, and the
        // negative ones (prmt with a sign-replicating selector gives 0xFF in
        // every negative byte)
        const int all = __dp4a(static_cast<int>(v.x), 0x01010101, __dp4a(static_cast<int>(v.y), 0x01010101, 0));
        const uint32_t nx = v.x & prmt(v.x, 0u, 0xBA98u), ny = v.y & prmt(v.y, 0u, 0xBA98u);
        const int ng = __dp4a(static_cast<int>(nx), 0x01010101, __dp4a(static_cast<int>(ny), 0x01010101, 0));
        neg += ng;
        pos += all - ng;
        abs += all - 2 * ng;
        // byte b ^ 0x80 is the weight plus 128 as an unsigned byte: the activation encoding gives the weight
        return cvt_u8x8(make_uint2(v.x ^ 0x80808080u, v.y ^ 0x80808080u));
    } else if constexpr (BITS == 4) {
        // 16 signed nibbles: sums from nibble sums (a negative nibble n stands for n - 16),
        // e4m3 codes by two prmt lookups (0..7 directly, 8..15 by magnitude 16 - n) plus the sign
        int all = 0, ng = 0;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const uint32_t x = h ? v.y : v.x;
            const int nneg = __popc(x & 0x88888888u);
            const uint32_t xm = x & (((x & 0x88888888u) >> 3) * 0xFu);  // the negative nibbles
            all += __dp4a(static_cast<int>((x & 0x0F0F0F0Fu) + ((x >> 4) & 0x0F0F0F0Fu)), 0x01010101, 0) - 16 * nneg;
            ng += __dp4a(static_cast<int>((xm & 0x0F0F0F0Fu) + ((xm >> 4) & 0x0F0F0F0Fu)), 0x01010101, 0) - 16 * nneg;
        }
        neg += ng;
        pos += all - ng;
        abs += all - 2 * ng;
        auto code4 = [](uint32_t q) {  // the low 16 bits of q: four signed nibbles -> four e4m3 bytes
            const uint32_t sgn = ((q & 0x8u) << 4) | ((q & 0x80u) << 8) | ((q & 0x800u) << 12) | ((q & 0x8000u) << 16);
            return prmt(0x44403800u, 0x4E4C4A48u, q) | prmt(0x4A4C4E50u, 0x38404448u, q ^ 0x8888u) | sgn;
        };
        return make_uint4(code4(v.x), code4(v.x >> 16), code4(v.y), code4(v.y >> 16));
    } else {
        // 16 signed crumbs (one word): sums from crumb sums (a negative crumb c stands for
        // c - 4), e4m3 codes by one 4-entry prmt lookup, in the converter's word order
        // (even channels, then odd, per half)
        const uint32_t x = v.x;
        const int nneg = __popc(x & 0xAAAAAAAAu);
        const uint32_t xm = x & (((x & 0xAAAAAAAAu) >> 1) * 0x3u);  // the negative crumbs
        const uint32_t c = (x & 0x33333333u) + ((x >> 2) & 0x33333333u);
        const uint32_t cm = (xm & 0x33333333u) + ((xm >> 2) & 0x33333333u);
        const int all = __dp4a(static_cast<int>((c & 0x0F0F0F0Fu) + ((c >> 4) & 0x0F0F0F0Fu)), 0x01010101, 0) - 4 * nneg;
        const int ng = __dp4a(static_cast<int>((cm & 0x0F0F0F0Fu) + ((cm >> 4) & 0x0F0F0F0Fu)), 0x01010101, 0) - 4 * nneg;
        neg += ng;
        pos += all - ng;
        abs += all - 2 * ng;
        constexpr uint32_t kCode = 0xB8C03800u;  // e4m3 of 0, 1, -2, -1 (crumbs 0..3)
        const uint32_t ev = x & 0x33333333u, od = (x >> 2) & 0x33333333u;
        return make_uint4(prmt(kCode, 0u, ev), prmt(kCode, 0u, od), prmt(kCode, 0u, ev >> 16), prmt(kCode, 0u, od >> 16));
    }
}

// What the MMA warp needs, made by warps 4-12 together: the B operand
// ([tap][K-chunk][NT rows][16 B]), the per-(channel, tap) absolute sums and
// the chunk count they allow, the MMA issue table, the pre-load operands and
// the slot layout.  The per-channel sums of positive and negative weights
// stay in shared memory for the compression records.
template <int BITS, int NT, bool FOLD>
__device__ __forceinline__ void prepare_filters(const WinArgs &a, uint8_t *smem, Misc *misc, uint64_t *w_full)
{
    constexpr int kGroupBytes = BITS == 8 ? 8 : 16 * BITS / 8;
    constexpr int kMaxX = BITS == 8 ? 128 : (1 << BITS) - 1;  // largest |staged activation|
    constexpr int kBatch = 2;                                   // items per thread whose loads go out together
    const int et = threadIdx.x - kPrepWarp0 * 32;
    int *tapabs = reinterpret_cast<int *>(smem + a.off_tap);    // [taps][NT]
    int *sums = tapabs + a.taps * NT;                           // [2][NT]: positive part, negative part
    for (int i = et; i < 2 * NT; i += kPrepThreads) sums[i] = 0;
    if (et == 0) misc->mask = ~0u;
    prep_sync();
    // item i: channel n = i % NT, tap i / NT; thread et takes items et, et + kPrepThreads, ...
    // K-chunks holding filter values, and packed bytes of one tap of one filter (a kernel
    // row's kw * c bytes when folded: they are contiguous in [m][kh][kw][c])
    const int cgroups = FOLD ? a.groups : a.c * BITS / 8 / kGroupBytes;
    const int items = a.taps * NT;
    const long long wrow = FOLD ? static_cast<long long>(a.kw) * a.c : static_cast<long long>(a.c) * BITS / 8;
    // the packed filters: the loader's shared-memory copy, or global memory
    const bool copied = a.wraw_bytes != 0;
    if (copied) mbar_wait_warp(w_full, 0, a.status);
    const uint8_t *wsrc = copied ? smem + a.off_wraw : a.w;
    for (int i0 = et; i0 < items; i0 += kBatch * kPrepThreads) {
        uint2 raw[kBatch][8];
#pragma unroll
        for (int b = 0; b < kBatch; ++b) {
            const int i = i0 + b * kPrepThreads, n = i % NT;
            const uint8_t *src = wsrc + (static_cast<long long>(n) * a.taps + i / NT) * wrow;
#pragma unroll
            for (int gq = 0; gq < 8; ++gq) {
                const bool has = i < items && n < a.m && gq < cgroups;
                if constexpr (BITS == 8 && FOLD) {
                    // bytes gq * 8 .. + 7 of the row's kw * c (unaligned; zero past its end)
                    uint32_t lo = 0, hi = 0;
                    for (int k = 0; has && k < 8 && gq * 8 + k < wrow; ++k) {
                        const uint32_t byte = src[gq * 8 + k];
                        if (k < 4) lo |= byte << (8 * k);
                        else hi |= byte << (8 * (k - 4));
                    }
                    raw[b][gq] = make_uint2(lo, hi);
                } else if (kGroupBytes == 8) {
                    const uint2 *q = reinterpret_cast<const uint2 *>(src + gq * 8);
                    raw[b][gq] = !has ? make_uint2(0u, 0u) : copied ? *q : __ldg(q);
                } else {
                    const uint32_t *q = reinterpret_cast<const uint32_t *>(src + gq * 4);
                    raw[b][gq] = make_uint2(!has ? 0u : copied ? *q : __ldg(q), 0u);
                }
            }
        }
#pragma unroll
        for (int b = 0; b < kBatch; ++b) {
            const int i = i0 + b * kPrepThreads;
            if (i >= items) break;
            const int n = i % NT, tap = i / NT;
            int pos = 0, neg = 0, abs = 0;
#pragma unroll
            for (int gq = 0; gq < 8; ++gq) {
                if (gq >= a.groups) break;
                // K-chunks past the channel count (and filters past m) stage +0
                const uint4 v = (n < a.m && gq < cgroups) ? filter_chunk<BITS>(raw[b][gq], pos, neg, abs)
                                                         : make_uint4(0u, 0u, 0u, 0u);
                *reinterpret_cast<uint4 *>(smem + a.off_b + ((tap * a.groups + gq) * NT + n) * 16) = v;
            }
            tapabs[tap * NT + n] = abs;
            if (n < a.m) {
                atomicAdd(&sums[n], pos);
                atomicAdd(&sums[NT + n], neg);
            }
        }
    }
    // Operands of the pre-load MMA (K-major, 8-row core matrices 128 bytes apart,
    // the second K-chunk 16 rows further): A rows {2048, 0, ...}, B rows {6144, 0, ...},
    // so every accumulator element becomes 2048 * 6144 = 1.5 * 2^23.
    {
        uint32_t *pre = reinterpret_cast<uint32_t *>(smem + a.off_pre);
        const int aw = 128 * 2 * 4, bw = NT * 2 * 4;  // 32-bit words: A (128 rows, 2 chunks), B (NT rows, 2 chunks)
        for (int i = et; i < aw + bw; i += kPrepThreads) {
            const bool is_a = i < aw;
            const int j = is_a ? i : i - aw;       // word within the operand
            const int rows = is_a ? 128 : NT;
            const bool first = j < rows * 4 && (j & 3) == 0;  // chunk 0, element 0 of a row
            pre[i] = first ? (is_a ? 0x6800u : 0x6E00u) : 0u;  // fp16 2048, 6144
        }
    }
    prep_sync();
    // Chunk counts c in [nch_min, c_force] whose even tap split has no empty
    // chunk and keeps every chunk of every channel exact; c_force = max(nch_min,
    // nch_max) holds by the planner's worst-case bound whatever the filters.
    const int c_force = max(a.nch_min, a.nch_max);
    if (et < NT) {
        uint32_t okmask = 0;
        for (int c = a.nch_min; c <= c_force; ++c) {
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
        okmask |= 1u << c_force;
        atomicAnd(&misc->mask, okmask);
    }
    prep_sync();
    const int nch = __ffs(static_cast<int>(misc->mask)) - 1;
    // K-split: a tile with a single accumulator (one strip, one chunk) and an
    // even k-step count alternates the k-steps of a tap between two
    // accumulators (each sums a subset of the chunk's products, so each is
    // exact where the chunk is), so that consecutive MMAs do not wait on each
    // other; the epilogue adds all nch * kx accumulators of a strip
    const int kx = (a.s * nch == 1 && a.ksteps % 2 == 0 && 2 * NT <= 256) ? 2 : 1;
    // The MMA issue order, one 8-byte entry per MMA: {A offset (16-byte units
    // within a stage) | accumulator column << 16, B offset}.  The accumulators
    // (chunk c, strip s) are independent and consecutive MMAs go to different
    // ones, so the tensor pipe does not wait on the previous MMA's accumulator:
    // the k-th step of every chunk and strip goes out together.  Thread et
    // writes the entries of step pair (jt, kk) = (et / ksteps, et % ksteps);
    // only the last chunk is shorter (last_len taps).
    const int ct = (a.taps + nch - 1) / nch, last_len = a.taps - (nch - 1) * ct;
    if (et < ct * a.ksteps) {
        const int jt = et / a.ksteps, kk = et - jt * a.ksteps;
        const int nj = jt < last_len ? nch : nch - 1;  // chunks with a tap at step jt
        const int before = jt * nch - max(0, jt - last_len);
        int u = a.s * (a.ksteps * before + kk * nj);
        uint2 *tab = reinterpret_cast<uint2 *>(smem + a.off_mtab);
        const uint32_t kstep_a = 2u * (a.chunk_stride >> 4), kstep_b = 2u * NT;
        for (int c = 0; c < nj; ++c) {
            const int tap = c * ct + jt, ti = tap / a.kwf, tj = tap - ti * a.kwf;
            for (int s = 0; s < a.s; ++s, ++u)
                tab[u] = make_uint2((static_cast<uint32_t>(ti * a.sp + tj) + kk * kstep_a + s * kCols) |
                                        (static_cast<uint32_t>((s * nch + c) * kx + kk % kx) * NT << 16),
                                    static_cast<uint32_t>(tap * a.groups) * NT + kk * kstep_b);
        }
    }
    if (et == 0) {
        const uint32_t cols = static_cast<uint32_t>(a.s * nch * kx * NT);
        misc->nch = static_cast<uint32_t>(nch * kx);
        misc->kx = static_cast<uint32_t>(kx);
        // the tap area's spare row carries both into a prepared image
        tapabs[(a.taps + 2) * NT] = nch * kx;
        tapabs[(a.taps + 2) * NT + 1] = kx;
        slot_layout<NT>(misc, cols);
        misc->nmma = static_cast<uint32_t>(a.s * a.taps * a.ksteps);
    }
    // B and the pre-load operands were written through the generic proxy; the
    // tensor cores read them through the async proxy
    fence_proxy_async_smem();
    // the MMA warp starts after this barrier: B, the table and the slot layout are complete
    tc_fence_before();
    prep_sync();
    tc_fence_after();
}

// The per-channel compression records (rec0 = {lam2, kappa, shift, mode},
// rec1 = {beta, ulo, uhi, lambda}, as in the tensor-core prep kernel, with
// acc + bias = s + beta for the raw chunk sum s) and the "all direct" flag of
// every 16 channels, made by the epilogue warps while the first tile's MMAs
// run (named barrier 2).
__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 2, %0;" ::"n"(kEpiWarps * 32) : "memory"); }

template <int BITS, int NT>
__device__ __forceinline__ void prepare_records(const WinArgs &a, uint8_t *smem, const Misc *misc)
{
    const int et = threadIdx.x - kEpiWarp0 * 32;
    const int *sums = reinterpret_cast<const int *>(smem + a.off_tap) + a.taps * NT;
    const int nch = static_cast<int>(misc->nch);
    int4 *rec0 = reinterpret_cast<int4 *>(smem + a.off_rec);
    int4 *rec1 = rec0 + NT;
    if (et < NT) {
        const int o = et;
        const long long off = BITS == 8 ? -128 : 0;  // staged activation = x + off
        const int s_w = sums[o] + sums[NT + o];
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
            const long long u0 = top * sums[NT + o] + b, u1 = top * sums[o] + b;
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
    // one "all direct" flag per 16-channel group
    uint8_t *gd = reinterpret_cast<uint8_t *>(rec1 + NT);
    if (et < NT / 16) {
        int all = 1;
        for (int k = 0; k < 16; ++k) all &= rec0[et * 16 + k].w == kModeDirect;
        gd[et] = static_cast<uint8_t>(all);
    }
    epi_sync();
}

// The prepared image: the loader's two bulk copies (B, then the tail) on w_full.
__device__ __forceinline__ void load_image(const WinArgs &a, uint8_t *smem, uint64_t *w_full)
{
    if ((threadIdx.x & 31) == 0) {
        mbar_arrive_expect_tx(w_full, a.b_bytes + a.tail_bytes);
        for (uint32_t off = 0; off < a.b_bytes; off += 32768u)
            bulk_g2s(smem + a.off_b + off, a.img + off, min(32768u, a.b_bytes - off), w_full);
        for (uint32_t off = 0; off < a.tail_bytes; off += 32768u)
            bulk_g2s(smem + a.off_rec + off, a.img + a.b_bytes + off, min(32768u, a.tail_bytes - off), w_full);
    }
    __syncwarp();
}

// Warps 4-12 with a prepared image: once it has landed, the slot layout
// follows from the accumulator count it carries.
template <int NT>
__device__ __forceinline__ void image_ready(const WinArgs &a, uint8_t *smem, Misc *misc, uint64_t *w_full)
{
    mbar_wait_warp(w_full, 0, a.status);
    if (threadIdx.x == kPrepWarp0 * 32) {
        const int *spare = reinterpret_cast<const int *>(smem + a.off_tap) + (a.taps + 2) * NT;
        const uint32_t nacc = static_cast<uint32_t>(spare[0]), cols = static_cast<uint32_t>(a.s) * nacc * NT;
        misc->nch = nacc;
        misc->kx = static_cast<uint32_t>(spare[1]);
        slot_layout<NT>(misc, cols);
        misc->nmma = static_cast<uint32_t>(a.s * a.taps * a.ksteps);
    }
    prep_sync();
}

// Warps 4-12 after the preparation: B and the tail out to the image (16-byte units).
__device__ __forceinline__ void store_image(const WinArgs &a, const uint8_t *smem)
{
    const int et = threadIdx.x - kPrepWarp0 * 32;
    for (uint32_t off = static_cast<uint32_t>(et) * 16u; off < a.b_bytes; off += kPrepThreads * 16u)
        *reinterpret_cast<uint4 *>(a.img_out + off) = *reinterpret_cast<const uint4 *>(smem + a.off_b + off);
    for (uint32_t off = static_cast<uint32_t>(et) * 16u; off < a.tail_bytes; off += kPrepThreads * 16u)
        *reinterpret_cast<uint4 *>(a.img_out + a.b_bytes + off) =
            *reinterpret_cast<const uint4 *>(smem + a.off_rec + off);
}

// ---------------------------------------------------------------- epilogue (warps 4-11)

// The integer sums of the chunks' bit patterns of EB consecutive columns of
// the tile's strips (chunk buffers `stride` columns apart, strip 1's buffers at
// a1).  With at most two chunks every load of the block is in flight before one
// wait.
template <int EB>
__device__ __forceinline__ void tmem_load(uint32_t addr, uint32_t (&v)[EB])
{
    if constexpr (EB >= 16) {
#pragma unroll
        for (int b0 = 0; b0 < EB; b0 += 16) tmem_ld16(addr + b0, *reinterpret_cast<uint32_t(*)[16]>(v + b0));
    } else if constexpr (EB == 8) {
        tmem_ld8(addr, *reinterpret_cast<uint32_t(*)[8]>(v));
    } else {
        tmem_ld4(addr, *reinterpret_cast<uint32_t(*)[4]>(v));
    }
}

// More than two chunks (long filters with large weights): one wait per chunk.
template <int EB>
__device__ __forceinline__ void drain_many(uint32_t a0, uint32_t a1, bool two, int nch, uint32_t stride, uint32_t (&v0)[EB],
                                        uint32_t (&v1)[EB])
{
#pragma unroll
    for (int k = 0; k < EB; ++k) v0[k] = v1[k] = 0;
#pragma unroll 1
    for (int c = 0; c < nch; ++c) {
        uint32_t t0[EB], t1[EB];
        tmem_load<EB>(a0 + c * stride, t0);
        if (two) tmem_load<EB>(a1 + c * stride, t1);
        tmem_wait_ld();
#pragma unroll
        for (int k = 0; k < EB; ++k) {
            v0[k] += t0[k];
            v1[k] += t1[k];
        }
    }
}

template <int EB>
__device__ __forceinline__ void drain_block(uint32_t a0, uint32_t a1, bool two, int nch, uint32_t stride,
                                            uint32_t (&v0)[EB], uint32_t (&v1)[EB])
{
    if (nch <= 2) {
        uint32_t t0[EB], t1[EB];
        tmem_load<EB>(a0, v0);
        if (nch == 2) tmem_load<EB>(a0 + stride, t0);
        if (two) {
            tmem_load<EB>(a1, v1);
            if (nch == 2) tmem_load<EB>(a1 + stride, t1);
        }
        tmem_wait_ld();
        if (nch == 2) {
#pragma unroll
            for (int k = 0; k < EB; ++k) {
                v0[k] += t0[k];
                v1[k] += t1[k];  // unused when !two
            }
        }
    } else {
        drain_many<EB>(a0, a1, two, nch, stride, v0, v1);
    }
}

// Q-bit packing of G compressed values (cvt.pack.sat: the clip of Sec. III-A
// fused with the packing of Sec. IV-A).
template <int BITS, int G>
__device__ __forceinline__ void pack_values(const int (&y)[G], uint32_t (&packed)[(G * BITS + 31) / 32])
{
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

// One block of EB output channels of one strip's pixel: packed Q-bit values,
// max-pooled over the 2x2 window when POOL (every lane shuffles), stored.
template <int BITS, int EB, bool POOL>
__device__ __forceinline__ void store_block(const int (&y)[EB], bool store, int valid, uint8_t *dst)
{
    uint32_t pk[(EB * BITS + 31) / 32];
    pack_values<BITS, EB>(y, pk);
    if constexpr (POOL) {
#pragma unroll
        for (int wd = 0; wd < (EB * BITS + 31) / 32; ++wd) {
            pk[wd] = max_fields<BITS>(pk[wd], __shfl_xor_sync(0xffffffffu, pk[wd], 1));
            pk[wd] = max_fields<BITS>(pk[wd], __shfl_xor_sync(0xffffffffu, pk[wd], 8));
        }
    }
    if (store) store_packed<BITS, EB>(pk, valid, dst);
}

// HB packed Q-bit values of one strip's pixel (whole words when HB * Q is a
// multiple of 32, else the low bits of one word): max-pooled over the 2x2
// window when POOL (every lane shuffles), stored.
template <int BITS, int HB, bool POOL>
__device__ __forceinline__ void store_words(uint32_t (&pk)[(HB * BITS + 31) / 32 < 1 ? 1 : (HB * BITS + 31) / 32],
                                            bool store, int valid, uint8_t *dst)
{
    if constexpr (POOL) {
#pragma unroll
        for (int wd = 0; wd < (HB * BITS + 31) / 32; ++wd) {
            pk[wd] = max_fields<BITS>(pk[wd], __shfl_xor_sync(0xffffffffu, pk[wd], 1));
            pk[wd] = max_fields<BITS>(pk[wd], __shfl_xor_sync(0xffffffffu, pk[wd], 8));
        }
    }
    if (store) store_packed<BITS, HB>(pk, valid, dst);
}

// Whether channel m's compression is in the direct form (flags per 16 channels).
__device__ __forceinline__ bool l_direct(const uint8_t *gdirect, int m) { return gdirect[m >> 4] != 0; }

// One tile's epilogue state for a warp: its TMEM columns, channels, output
// pixels and whether the direct form with one shift covers all its channels.
template <int NT>
struct EpiTile {
    uint32_t base, strip1;
    bool two;
    int nch, col0, lane;
    bool direct_all, one_shift;
    uint32_t shift;
    const int4 *rec0, *rec1;
    uint8_t *dst[2];
    bool store[2];
    uint64_t *acc_empty;
    bool tmem_cst;     // lam2 and kappa of the block's channels come from TMEM with the accumulators
    uint32_t cst_addr; // TMEM address of lam2 of channel col0 in this warp's lanes (kappa NT columns on)
};

// The tile's columns in blocks of HB: the loads of a block (NCH accumulators
// per strip, 0 = any count, one wait per accumulator), the slot released
// after the last block's loads, then compression, packing and stores (HB
// values of a pixel are HB * Q / 8 contiguous bytes).
template <int BITS, int NT, bool POOL, int HB, int NCH>
__device__ __forceinline__ void epi_tile(const WinArgs &a, const EpiTile<NT> &e, const uint32_t (&my_lam2)[2],
                                         const uint32_t (&my_kap)[2], const uint32_t (&my_sh)[2])
{
    constexpr int CW = NT / 2;
#pragma unroll 1
    for (int k0 = 0; k0 < CW; k0 += HB) {
        uint32_t v0[HB], v1[HB], cl[HB], ck[HB];  // accumulators; lam2 and kappa when tmem_cst
        if constexpr (NCH == 0) {
            drain_many<HB>(e.base + k0, e.base + e.strip1 + k0, e.two, e.nch, NT, v0, v1);
        } else {
            uint32_t t0[NCH == 2 ? HB : 1], t1[NCH == 2 ? HB : 1];
            if (e.tmem_cst) {
                tmem_load<HB>(e.cst_addr + k0, cl);
                tmem_load<HB>(e.cst_addr + NT + k0, ck);
            }
            tmem_load<HB>(e.base + k0, v0);
            if constexpr (NCH == 2) tmem_load<HB>(e.base + k0 + NT, t0);
            if (e.two) {
                tmem_load<HB>(e.base + e.strip1 + k0, v1);
                if constexpr (NCH == 2) tmem_load<HB>(e.base + e.strip1 + k0 + NT, t1);
            }
            tmem_wait_ld();
#pragma unroll
            for (int k = 0; k < HB; ++k) {
                asm volatile("" : "+r"(v0[k]), "+r"(v1[k]), "+r"(cl[k]), "+r"(ck[k]));  // uses stay after the wait
                if constexpr (NCH == 2) {
                    asm volatile("" : "+r"(t0[k]), "+r"(t1[k]));
                    v0[k] += t0[k];
                    v1[k] += t1[k];  // unused when !two
                }
            }
        }
        if (k0 + HB >= CW) {  // the slot's last columns are read: give it back first
            tc_fence_before();
            __syncwarp();
            if (e.lane == 0) mbar_arrive(e.acc_empty);
        }
        const int m0 = e.col0 + k0;
        const int valid = a.m - m0;  // same for the whole warp
        if (valid <= 0) continue;
        // groups of 8 channels: their constants, both strips' values, packed at once
        constexpr int kG = HB < (BITS == 2 ? 16 : 8) ? HB : (BITS == 2 ? 16 : 8);  // a whole number of words
        constexpr int kGW = (kG * BITS + 31) / 32;  // packed words per group
        uint32_t pk0[HB / kG * kGW], pk1[HB / kG * kGW];
#pragma unroll
        for (int g0 = 0; g0 < HB; g0 += kG) {
            int y0[kG], y1[kG];
            if (NCH != 0 && e.tmem_cst) {
                // direct form, one shift: the constants arrived with the accumulators
#pragma unroll
                for (int k = 0; k < kG; ++k) {
                    y0[k] = static_cast<int32_t>(v0[g0 + k] * ck[g0 + k] + cl[g0 + k]) >> e.shift;
                    y1[k] = static_cast<int32_t>(v1[g0 + k] * ck[g0 + k] + cl[g0 + k]) >> e.shift;
                }
            } else if (e.direct_all) {
                // direct channels: ((s * kappa + lam2) mod 2^32) >> shift is exact (see the records);
                // the constants of channel col0 + k0 + k sit in lane (k0 + k) % 32 of set (k0 + k) / 32
#pragma unroll
                for (int k = 0; k < kG; ++k) {
                    const int c = k0 + g0 + k, set = c >= 32 ? 1 : 0;
                    const uint32_t lam2 = __shfl_sync(0xffffffffu, set ? my_lam2[1] : my_lam2[0], c & 31);
                    const uint32_t kap = __shfl_sync(0xffffffffu, set ? my_kap[1] : my_kap[0], c & 31);
                    const uint32_t sh =
                        e.one_shift ? e.shift : __shfl_sync(0xffffffffu, set ? my_sh[1] : my_sh[0], c & 31);
                    y0[k] = static_cast<int32_t>(v0[g0 + k] * kap + lam2) >> sh;
                    y1[k] = static_cast<int32_t>(v1[g0 + k] * kap + lam2) >> sh;
                }
            } else {
#pragma unroll
                for (int k = 0; k < kG; ++k) {
                    const int4 r0 = e.rec0[m0 + g0 + k], r1 = e.rec1[m0 + g0 + k];
                    y0[k] = static_cast<int>(compress_slow(v0[g0 + k], r0, r1, (1u << BITS) - 1u));
                    y1[k] = e.two ? static_cast<int>(compress_slow(v1[g0 + k], r0, r1, (1u << BITS) - 1u)) : 0;
                }
            }
            pack_values<BITS, kG>(y0, *reinterpret_cast<uint32_t(*)[kGW]>(pk0 + g0 / kG * kGW));
            pack_values<BITS, kG>(y1, *reinterpret_cast<uint32_t(*)[kGW]>(pk1 + g0 / kG * kGW));
        }
        store_words<BITS, HB, POOL>(pk0, e.store[0], valid, e.dst[0] + m0 * BITS / 8);
        if (e.two) store_words<BITS, HB, POOL>(pk1, e.store[1], valid, e.dst[1] + m0 * BITS / 8);
    }
}

template <int BITS, int NT, bool POOL>
__device__ __forceinline__ void epilogue_role(const WinArgs &a, uint8_t *smem, uint64_t *acc_full, uint64_t *acc_empty,
                                              const Misc *misc)
{
    constexpr int CW = NT / 2;             // columns of this warp
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quarter = warp & 3, half = (warp - kEpiWarp0) >> 2;
    const int row = quarter * 32 + lane;  // tile row of a strip: 8 * (output row) + column
    const int col0 = half * CW;
    const uint32_t tmem = misc->tmem;
    const int nch = static_cast<int>(misc->nch), nslots = static_cast<int>(misc->nslots);
    const uint32_t slot_cols = misc->slot_cols;
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + col0;
    const int4 *rec0 = reinterpret_cast<const int4 *>(smem + a.off_rec);
    const int4 *rec1 = rec0 + NT;
    const uint8_t *gdirect = reinterpret_cast<const uint8_t *>(rec1 + NT);
    const int out_row_bytes = a.m * BITS / 8;
    const bool two = a.s == 2;
    // This warp's channels are fixed: lane l keeps channel col0 + l's direct-form
    // constants in registers and broadcasts them with shuffles, so the inner loop
    // touches no shared memory (the tensor cores keep it busy with operand reads).
    constexpr int LW = CW < 32 ? CW : 32;  // channels per register set
    uint32_t my_lam2[2], my_kap[2], my_sh[2];
    bool direct_all = true;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        const int m = col0 + (r * 32 < CW ? r * 32 : 0) + lane % LW;
        const int4 rec = rec0[m];
        my_lam2[r] = static_cast<uint32_t>(rec.x);
        my_kap[r] = static_cast<uint32_t>(rec.y);
        my_sh[r] = static_cast<uint32_t>(rec.z);
        direct_all = __all_sync(0xffffffffu, l_direct(gdirect, m)) && direct_all;
    }
    // one shift for all of this warp's channels: the common case, one shuffle less per value
    const uint32_t shift = __shfl_sync(0xffffffffu, my_sh[0], 0);
    const bool one_shift = __all_sync(0xffffffffu, my_sh[0] == shift && my_sh[1] == shift);
    const uint32_t strip1 = static_cast<uint32_t>(nch) * NT;  // columns from strip 0's buffers to strip 1's
    int *const status = a.status;
    // The direct-form constants of this warp's channels, one row per lane of its
    // quarter (all rows alike): the block loop reads them with the accumulators
    // instead of broadcasting them lane to lane (shuffles queue behind the
    // tensor cores' shared-memory reads).
    const uint32_t cst = misc->cst;
    const bool tmem_cst = cst != ~0u && direct_all && one_shift;
    const uint32_t cst_addr = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + cst + col0;
    if (tmem_cst) {
#pragma unroll 1
        for (int j = 0; j < CW; j += 16) {
            uint32_t l[16], kp[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) {
                const int4 r = rec0[col0 + j + k];
                l[k] = static_cast<uint32_t>(r.x);
                kp[k] = static_cast<uint32_t>(r.y);
            }
            tmem_st16(cst_addr + j, l);
            tmem_st16(cst_addr + NT + j, kp);
        }
        tmem_wait_st();
    }

    const int oyr = row >> 3, oxr = row & 7;
    for (int i = 0, t = blockIdx.x; t < a.total_tiles; ++i, t += gridDim.x) {
        const int slot = i % nslots;
        const Geo g = geo_of(a, t);
        if (!mbar_wait_warp(&acc_full[slot], (i / nslots) & 1, status)) return;
        tc_fence_after();
        const int oy = g.oy0 + oyr;
        // where strip s's pixel of this lane goes: its output row, or its pooled pixel
        uint8_t *dst[2];
        bool store[2];
#pragma unroll
        for (int s = 0; s < 2; ++s) {
            const int ox = g.ox0 + s * kCols + oxr;
            if constexpr (POOL) {
                // pooled pixel (oy/2, ox/2) is the 2x2 window of lanes L, L^1, L^8, L^9; its top-left lane stores
                store[s] = (row & 9) == 0 && (oy >> 1) < a.pool_oh && (ox >> 1) < a.pool_ow;
                dst[s] = a.y + ((static_cast<long long>(g.img) * a.pool_oh + (oy >> 1)) * a.pool_ow + (ox >> 1)) *
                                   out_row_bytes;
            } else {
                store[s] = oy < a.oh && ox < a.ow;
                dst[s] = a.y + ((static_cast<long long>(g.img) * a.oh + oy) * a.ow + ox) * out_row_bytes;
            }
            store[s] = store[s] && (s == 0 || two);
        }
        const uint32_t base = lane_addr + slot * slot_cols;
        const EpiTile<NT> et{base,     strip1,  two,   nch,  col0,     lane,
                             direct_all, one_shift, shift, rec0, rec1,  {dst[0], dst[1]},
                             {store[0], store[1]}, &acc_empty[slot], tmem_cst, cst_addr};
        // every load of a block of 8 columns (both strips' accumulators and, with
        // tmem_cst, the constants) goes out before one wait; more than two
        // accumulators per strip: one wait per accumulator
        if (nch == 1) epi_tile<BITS, NT, POOL, (CW < 8 ? CW : 8), 1>(a, et, my_lam2, my_kap, my_sh);
        else if (nch == 2) epi_tile<BITS, NT, POOL, (CW < 8 ? CW : 8), 2>(a, et, my_lam2, my_kap, my_sh);
        else epi_tile<BITS, NT, POOL, (CW < 8 ? CW : 8), 0>(a, et, my_lam2, my_kap, my_sh);
    }
}

// ---------------------------------------------------------------- the kernel

template <int BITS, int NT, bool POOL, bool FOLD>
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
    uint64_t *done = acc_empty + kMaxSlots;
    uint64_t *w_full = done + 1;
    Misc *misc = reinterpret_cast<Misc *>(w_full + 2);  // (one spare barrier slot)
    const int warp = threadIdx.x >> 5;
    // Programmatic dependent launch: the next kernel in the stream may launch
    // now; its blocks take each SM as this kernel's block there exits, and do
    // their setup while the rest of this grid finishes.  A launch that writes
    // a prepared image (img_out) does not: its successor starts after it ends,
    // so a convolving launch may read its image before waiting on its
    // predecessor (every image was written by an earlier, finished launch).
    if (a.img_out == nullptr) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

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
            mbar_init(done, 1);
            mbar_init(w_full, 1);
            fence_mbar_init();
        }
        __syncwarp();
        tmem_alloc(&misc->tmem, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // the prepared image comes from a finished launch: its copy may start now
    if (warp == kLoadWarp && a.img) load_image(a, smem, w_full);
    // nothing above reads other global memory: from here on, everything the
    // previous kernel in the stream wrote is visible
    asm volatile("griddepcontrol.wait;" ::: "memory");

    // Each warp takes its role.  The loader copies the filters (or the
    // prepared image), then streams the windows; the converters stage windows
    // from the start; the epilogue warps and the MMA warp first prepare the
    // filters together (or wait for the image).  With img_out the block only
    // prepares the filters and writes the image.
    const bool convolve = a.img_out == nullptr;
    if (warp < kConvWarps) {
        if (convolve) {
            if constexpr (BITS == 8 && FOLD) converter_fold(a, smem, raw_full, raw_empty, a_full, a_empty);
            else converter_role<BITS>(a, smem, raw_full, raw_empty, a_full, a_empty);
        }
    } else if (warp == kLoadWarp) {
        if (!a.img) load_filters(a, smem, w_full);
        if (convolve) {
            LoadState ld{0, 0, static_cast<int>(blockIdx.x), 0u};
            load_windows(a, smem, raw_full, raw_empty, ld, a.total_tiles);
            load_drain(a, raw_full, w_full, ld);
        }
    } else {
        if (a.img) {
            image_ready<NT>(a, smem, misc, w_full);
        } else {
            prepare_filters<BITS, NT, FOLD>(a, smem, misc, w_full);
        }
        if (warp == kMmaWarp) {
            if (convolve) mma_role<NT, BITS != 8>(a, smem, a_full, a_empty, acc_full, acc_empty, done, misc);
        } else {
            // all slots start free (the MMA warp writes each accumulator's pre-load)
            if (convolve && (threadIdx.x & 31) == 0)
                for (uint32_t slot = 0; slot < misc->nslots; ++slot) mbar_arrive(&acc_empty[slot]);
            if (!a.img) prepare_records<BITS, NT>(a, smem, misc);
            if (convolve) epilogue_role<BITS, NT, POOL>(a, smem, acc_full, acc_empty, misc);
        }
        if (!convolve) {
            prep_sync();
            store_image(a, smem);
        }
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
