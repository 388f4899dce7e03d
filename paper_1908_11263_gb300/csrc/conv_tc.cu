// Quantized HWC convolution as an implicit GEMM on the sm_103a tensor cores.
//
// What it computes (Sec. III-B, Eq. 6; Sec. III-A, Eq. 2 and the scale-and-clamp
// compression): for every output pixel p and channel o,
//   acc = dot(W(o), im2col(p))                     exact integer, int32
//   y   = clip(floor(((acc + bias_o) * kappa_o + lambda_o) / 2^shift_o), 0, 2^Q - 1)
//
// GEMM view: rows = 128 consecutive output pixels of one image (MMA M = 128),
// columns = output channels (MMA N = NT), K = kh * kw * c (tap-major, channel
// minor: the im2col order of Eq. 6).  Stride 1.
//
// Exactness on fp16 tensor cores.  GB300 has no integer tcgen05 MMA, so the
// integers are embedded exactly in fp16 and multiplied with fp32 accumulation
// (kind::f16):
//   * INT-8: activations are staged as x - 128 in [-128, 127], weights as
//     themselves; |product| <= 2^14.  INT-4 / INT-2: activations are staged as
//     x + 1024 (an fp16 with the integer in its low mantissa bits), weights as
//     themselves.  All these values and products are exact in fp16 / fp32.
//   * Each accumulator is pre-loaded with 1.5 * 2^23 (bits 0x4B400000) and
//     receives at most 2^22 / max|product| products, so every partial sum stays
//     in [2^23, 2^24], where fp32 holds every integer; the final bit pattern
//     minus 0x4B400000 is the chunk's integer sum.  Longer K is split into
//     several chunks, summed as integers in the epilogue.
//   * The offsets are removed exactly with a per-channel constant (128 * sum(W)
//     or -1024 * sum(W)) folded in by the prep kernel.
//
// im2col without copies.  For stride 1, the A operand of tap (i, j) is the
// staged input shifted by i rows and j columns.  The stage keeps one copy of
// the input window per horizontal tap j (padding columns pre-filled with the
// encoded zero), stored as [copy j][8-channel chunk][position][8 x fp16].  Rows
// of A are then 16 bytes apart for every tap, so the tap (i, j) operand is the
// same no-swizzle K-major layout started i * ow positions later: one
// shared-memory descriptor per MMA, no im2col buffer.  Descriptor offsets of
// every (tap, k-step) are tabulated once per CTA, so issuing an MMA costs a
// table load and two additions.
//
// Data movement per tile: one bulk (TMA) copy brings the tile's input rows
// (all channels, HBM -> shared memory); converter warps turn each element
// into fp16 once and store it into the kw copies; the filters are either
// resident in shared memory or streamed per (channel slab, tap) by bulk
// copies.  Accumulators form a ring of up to four TMEM buffers, so the MMAs of
// the next tile run while the epilogue compresses the current one.
//
// Warp roles (one persistent CTA per SM, 16 warps):
//   warps 0-3   converters: raw window -> staged fp16 (or e4m3) operand
//   warps 4-11  epilogue, two per TMEM lane quarter (one per column half):
//               TMEM -> registers, integer sum of chunks, compression, Q-bit
//               packing, store
//   warp 12     MMA issue (the warp runs converged; an elected lane issues)
//   warp 13     bulk copies of input rows (lane 0 issues)
//   warp 14     bulk copies of filters (lane 0 issues)
//   warp 15     second MMA issuer, taking alternate tiles, when one resident
//               filter set serves the whole kernel
// Every wait is bounded; on a timeout the kernel records QNN_ETIMEOUT in the
// status word, stops its work, lets its copies and MMAs drain and frees TMEM.
#include <cuda_fp16.h>

#include <algorithm>
#include <mutex>

#include "conv_common.cuh"
#include "device.cuh"
#include "internal.h"

namespace qnn {
namespace {

constexpr int kTileM = 128;
// Strip tiles: 16 output rows x 8 output columns (see the planner).
constexpr int kStripRows = 16, kStripCols = 8;
// Warp roles: converters 0-3, epilogue 4-11 (two warps per TMEM lane
// quarter, one per column half), MMA issuer 12, input-row loader 13, filter
// loader 14, second MMA issuer 15 (takes alternate tiles when the whole
// kernel uses one resident filter set).
constexpr int kConvWarps = 4, kEpiWarps = 8;
constexpr int kMmaWarp = 12, kRawWarp = 13, kBWarp = 14, kMmaWarp2 = 15;
constexpr int kWarps = 16;
constexpr int kThreads = kWarps * 32;
constexpr int kMaxSmem = 232448;          // 227 KB opt-in dynamic shared memory per block
constexpr uint32_t kCopyChunk = 32768;    // bytes per bulk copy instruction
constexpr int kMaxAccGroups = 4;
constexpr int kMaxTaps = 64;  // kh * kw limit of the tensor-core kernel

// Per-A-stage record the converter publishes with a_full for the MMA warp:
// bits 0-15 hold the tile's first pixel column d0, and two flags mark the first
// and last tile of a run that shares one resident filter set.
constexpr uint32_t kInfoRunStart = 1u << 30, kInfoRunEnd = 1u << 31;
constexpr int kMaxStages = 4;

struct TcArgs {
    const uint8_t *x;
    uint8_t *y;
    const uint8_t *wpack;  // fp16 filters [n_ntiles][k_pad/8][nt][8]
    const int4 *chan;      // [2][n_ntiles * nt] compression records
    int n, h, w, c, m, kh, kw, ph, pw, oh, ow;
    int c_pad, cs, nslab, log2_groups;
    int n_ntiles, tiles_per_img;
    int total_tiles;
    int rows_max, p_alloc;
    int stages, raw_stages, b_stages, b_resident;
    int mmas_per_tile, chunk_mmas, nchunks, grp_chunks, ngroups, nsg;
    uint32_t row_bytes, raw_bytes, b_bytes, b_tile_bytes, copy_bytes, stage_bytes, chunk_stride;
    uint32_t off_raw, off_stages, off_chan, off_bar, off_rec;
    uint32_t tmem_cols;
    int *status;
    FastDiv fd_per_nt, fd_tpi, fd_ow, fd_w;  // n * tiles_per_img, tiles_per_img, ow, pixels per staged row
    int strip;                                // tiles are 16 x 8 strips staged as one padded window
    int ncb, sp;                              // strips: column blocks per image, window width (pixels)
    int ncol_w;                               // pixels per staged row: w (row tiles) or sp (strips)
    uint32_t a_sbo;                           // A descriptor: bytes between 8-row core-matrix groups
    uint32_t d0_mask;                         // stage-word bits the MMA adds to the A address
    FastDiv fd_ncb;
    int conv_fast;                            // converter fast path (see ConvItem)
    int pool, pool_oh, pool_ow;               // fused 2x2/2 max-pool and its output height, width
    int fp8;                                  // e4m3 staging and kind::f8f6f4 MMAs (INT-4/INT-2)
    int kch;                                  // channels per 16-byte K-chunk: 8 (fp16) or 16 (e4m3)
    int mma_warps;                            // 2: warps 12 and 15 issue alternate tiles
    const int32_t *thr;                       // staircase thresholds in the workspace, or null
    uint32_t off_thr;                         // their shared-memory copy
    uint32_t tap_a16[kMaxTaps];  // per tap (i, j): A offset j*copy + i*ow positions, in 16-byte units
};

// Geometry of one tile: 128 consecutive output pixels of image `img` (row
// tiles), or output rows oy_a .. oy_a + 15 by columns d0 .. d0 + 7 (strips).
struct TileGeo {
    int nt, img, ti;
    int oy_a;   // first output row touched
    int d0;     // column of the first pixel within that row
    int rows;   // staged input rows (window height)
    int r_lo;   // staged rows [r_lo, r_hi) lie inside the image
    int r_hi;
};

__device__ __forceinline__ TileGeo tile_geo(const TcArgs &a, int t)
{
    const int per_nt = a.n * a.tiles_per_img;  // total tiles < 2^31 (checked by the planner)
    TileGeo g;
    g.nt = fdiv(t, a.fd_per_nt);
    const int rem = t - g.nt * per_nt;
    g.img = fdiv(rem, a.fd_tpi);
    g.ti = rem - g.img * a.tiles_per_img;
    if (a.strip) {
        const int rb = fdiv(g.ti, a.fd_ncb);
        g.oy_a = rb * kStripRows;
        g.d0 = (g.ti - rb * a.ncb) * kStripCols;
        g.rows = min(a.rows_max, a.oh - g.oy_a + a.kh - 1);
    } else {
        const int p0 = g.ti * kTileM;
        g.oy_a = fdiv(p0, a.fd_ow);
        g.d0 = p0 - g.oy_a * a.ow;
        const int out_rows = min(fdiv(g.d0 + kTileM + a.ow - 1, a.fd_ow), a.oh - g.oy_a);
        g.rows = min(a.rows_max, out_rows + a.kh - 1);
    }
    const int iy0 = g.oy_a - a.ph;
    g.r_lo = min(g.rows, max(0, -iy0));
    g.r_hi = max(g.r_lo, min(g.rows, a.h - iy0));
    return g;
}

__device__ __forceinline__ int tile_nt(const TcArgs &a, int t) { return fdiv(t, a.fd_per_nt); }

__device__ __forceinline__ bool nt_run_starts(const TcArgs &a, int t)
{
    return t == static_cast<int>(blockIdx.x) || tile_nt(a, t - gridDim.x) != tile_nt(a, t);
}

__device__ __forceinline__ bool nt_run_ends(const TcArgs &a, int t)
{
    const int nx = t + gridDim.x;
    return nx >= a.total_tiles || tile_nt(a, nx) != tile_nt(a, t);
}

// Warp-converged bounded wait (all lanes poll; the result is warp-uniform).
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, int *status)
{
    return mbar_wait_warp(bar, parity, status);
}

// ---------------------------------------------------------------- u8 / sub-byte -> fp16 (8 channels)

// Any channel count: channels c0.. of the pixel whose packed data starts at element e0 of `src`.
template <int BITS>
__device__ __noinline__ uint4 cvt_generic(const uint8_t *src, int e0, int c0, int c)
{
    uint16_t hv[8];
#pragma unroll
    for (int s = 0; s < 8; ++s) {
        const int ch = c0 + (BITS == 8 ? s : ((s & 1) ? 4 + (s >> 1) : (s >> 1)));
        int v = 0;
        if (ch < c) {
            const int e = e0 + ch;
            constexpr int per = 8 / BITS;
            v = (src[e / per] >> ((e % per) * BITS)) & ((1 << BITS) - 1);
        }
        v += (BITS == 8) ? -128 : 1024;
        hv[s] = __half_as_ushort(__int2half_rn(v));
    }
    uint4 r;
    r.x = hv[0] | (static_cast<uint32_t>(hv[1]) << 16);
    r.y = hv[2] | (static_cast<uint32_t>(hv[3]) << 16);
    r.z = hv[4] | (static_cast<uint32_t>(hv[5]) << 16);
    r.w = hv[6] | (static_cast<uint32_t>(hv[7]) << 16);
    return r;
}

// ---------------------------------------------------------------- converters (warps 0-3)

// Which column items a converter thread owns, fixed for the whole kernel.  A
// column item is one (8-channel group gq, pixel x) pair of a staged row, x
// fastest, so consecutive threads store consecutive 16-byte positions.  When a
// row has fewer than 128 items the 128 threads split into `nphase` row phases.
struct ConvMap {
    int ci0, cstep;  // first column item and stride
    int rp, nphase;  // first row and row stride
};

__device__ __forceinline__ ConvMap conv_map(int ncol)
{
    const int t = threadIdx.x;  // 0..127
    ConvMap m;
    if (ncol <= 128) {
        m.nphase = 128 / ncol;
        m.rp = t / ncol;
        m.ci0 = m.rp < m.nphase ? t - m.rp * ncol : ncol;  // threads past the last phase stay idle
        m.cstep = ncol;
        if (m.rp >= m.nphase) m.rp = 0;
    } else {
        m.nphase = 1;
        m.rp = 0;
        m.ci0 = t;
        m.cstep = 128;
    }
    return m;
}

// Loads 8 channels of one pixel from a staged raw row and widens them to the
// staged fp16 encoding (padding value when `ok` is false).
template <int BITS>
__device__ __forceinline__ uint4 load_cvt(const uint8_t *p, bool ok, bool vec, const uint8_t *row, int e0, int c0, int c)
{
    const uint32_t padv = pad_half2<BITS>();
    uint4 v = make_uint4(padv, padv, padv, padv);
    if (ok) {
        if (!vec && BITS == 8) {
            // C not a multiple of 8: the group's channels byte by byte (zero past C;
            // padded channels meet zero weights)
            uint32_t b[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) b[k] = c0 + k < c ? row[e0 + c0 + k] : 0u;
            v = cvt_u8x8(make_uint2(b[0] | b[1] << 8 | b[2] << 16 | b[3] << 24, b[4] | b[5] << 8 | b[6] << 16 | b[7] << 24));
        } else if (!vec) {
            v = cvt_generic<BITS>(row, e0, c0, c);
        } else if (BITS == 8) {
            v = cvt_u8x8(*reinterpret_cast<const uint2 *>(p));
        } else if (BITS == 4) {
            v = cvt_u4x8(*reinterpret_cast<const uint32_t *>(p));
        } else {
            v = cvt_u2x8(*reinterpret_cast<const uint16_t *>(p));
        }
    }
    return v;
}

// Stores one converted pixel into the copies j < NJ whose predicate is set
// (copy j holds the pixel one position further left per j).
template <int NJ>
__device__ __forceinline__ void store_copies(uint8_t *dst, uint32_t jstep, const bool (&pj)[5], const uint4 &v)
{
#pragma unroll
    for (int j = 0; j < NJ; ++j)
        if (pj[j]) *reinterpret_cast<uint4 *>(dst + j * jstep) = v;
}

// Rows rp, rp + nph, ... < rows of one column item, kRowsPerPass rows per pass:
// all of a pass's loads are in flight together before its stores, and rows
// past the window are predicated off.  The benchmark-shaped tiles (ten staged
// rows, two row phases) take a single pass.
constexpr int kRowsPerPass = 6;

template <int BITS, int NJ>
__device__ __forceinline__ void convert_rows(const uint8_t *src, uint8_t *dst, int rp, int nph, int rows, int r_lo,
                                             int r_hi, bool has_data, bool vec, uint32_t row_bytes, uint32_t row_out,
                                             uint32_t jstep, const bool (&pj)[5], const uint8_t *raw, int e0, int c0,
                                             int c)
{
    // src / dst point at row rp; src is only dereferenced for rows inside the image
    const uint32_t src_step = row_bytes * nph, dst_step = row_out * nph;
    for (int r = rp; r < rows; r += kRowsPerPass * nph) {
        uint4 v[kRowsPerPass];
#pragma unroll
        for (int u = 0; u < kRowsPerPass; ++u) {
            const int rr = r + u * nph;
            const bool ok = rr < rows && rr >= r_lo && rr < r_hi && has_data;
            v[u] = load_cvt<BITS>(src + u * src_step, ok, vec, raw + (rr - r_lo) * row_bytes, e0, c0, c);
        }
#pragma unroll
        for (int u = 0; u < kRowsPerPass; ++u)
            if (r + u * nph < rows) store_copies<NJ>(dst + u * dst_step, jstep, pj, v[u]);
        src += kRowsPerPass * src_step;
        dst += kRowsPerPass * dst_step;
    }
}

// One (tile, channel slab): staged raw rows -> kw fp16 copies, where copy j
// holds input pixel (r, ox + j - pw) at position r * ow + ox.  Each thread owns
// fixed column items (see conv_map) and walks the tile's staged rows for them:
// per row one load, one conversion and one store per copy that holds the pixel.
// Rows outside the image store the encoded zero.  Positions of columns that
// fall outside the image are never written (they keep the encoded zero
// written at kernel start).
template <int BITS>
__device__ __forceinline__ void convert_stage(const TcArgs &a, const uint8_t *raw, uint8_t *stage, const TileGeo &g,
                                              int slab, bool vec, const ConvMap &mp)
{
    const int ncol = a.ncol_w << a.log2_groups;
    const int cb = a.c * BITS / 8;  // packed bytes per pixel
    if (a.strip) {
        // One padded window, sp pixels wide: window pixel px of row r holds input
        // pixel (r, d0 - pw + px) at position r * sp + px, the encoded zero where
        // that pixel lies outside the image.  Every position of the tile's rows
        // is written, so no copy and no state from earlier tiles is involved.
        const uint32_t row_out = static_cast<uint32_t>(a.sp) * 16;
        const bool pone[5] = {true, false, false, false, false};
        for (int ci = mp.ci0; ci < ncol; ci += mp.cstep) {
            const int gq = fdiv(ci, a.fd_w);
            const int px = ci - gq * a.sp;
            const int c0 = slab * a.cs + gq * 8;
            if (c0 >= a.c) continue;  // a group wholly past C keeps the encoded zero
            const int ix = g.d0 - a.pw + px;
            const bool col_ok = ix >= 0 && ix < a.w;
            const int rp = mp.rp;
            const uint8_t *src = raw + (rp - g.r_lo) * static_cast<int>(a.row_bytes) + ix * cb + c0 * BITS / 8;
            uint8_t *dst = stage + gq * a.chunk_stride + (rp * a.sp + px) * 16;
            convert_rows<BITS, 1>(src, dst, rp, mp.nphase, g.rows, g.r_lo, g.r_hi, col_ok, vec, a.row_bytes, row_out,
                                  0u, pone, raw, ix * a.c, c0, a.c);
        }
        return;
    }
    const uint32_t jstep = a.copy_bytes - 16;
    const uint32_t row_out = static_cast<uint32_t>(a.ow) * 16;
    for (int ci = mp.ci0; ci < ncol; ci += mp.cstep) {
        const int gq = fdiv(ci, a.fd_w);
        const int x = ci - gq * a.w;
        const int c0 = slab * a.cs + gq * 8;
        // a group wholly past C keeps the encoded zero written at kernel start
        if (c0 >= a.c) continue;
        // copies j in [jlo, jhi] hold this pixel (their column x + pw - j lies in [0, ow))
        const int jlo = max(0, x + a.pw - a.ow + 1), jhi = min(a.kw - 1, x + a.pw);
        bool pj[5];
#pragma unroll
        for (int j = 0; j < 5; ++j) pj[j] = j >= jlo && j <= jhi;
        const int rp = mp.rp;
        const uint8_t *src = raw + (rp - g.r_lo) * static_cast<int>(a.row_bytes) + x * cb + c0 * BITS / 8;
        uint8_t *dst = stage + gq * a.chunk_stride + (x + a.pw) * 16 + rp * row_out;
        if (a.kw <= 3)
            convert_rows<BITS, 3>(src, dst, rp, mp.nphase, g.rows, g.r_lo, g.r_hi, c0 < a.c, vec, a.row_bytes, row_out,
                                  jstep, pj, raw, x * a.c, c0, a.c);
        else if (a.kw <= 5)
            convert_rows<BITS, 5>(src, dst, rp, mp.nphase, g.rows, g.r_lo, g.r_hi, c0 < a.c, vec, a.row_bytes, row_out,
                                  jstep, pj, raw, x * a.c, c0, a.c);
        else
            for (int r = rp; r < g.rows; r += mp.nphase) {  // wide kernels: any kw
                const bool ok = r >= g.r_lo && r < g.r_hi && c0 < a.c;
                const uint4 v = load_cvt<BITS>(raw + (r - g.r_lo) * static_cast<int>(a.row_bytes) + x * cb + c0 * BITS / 8,
                                               ok, vec, raw + (r - g.r_lo) * static_cast<int>(a.row_bytes), x * a.c, c0, a.c);
                uint8_t *d = stage + gq * a.chunk_stride + (x + a.pw) * 16 + r * row_out;
                for (int j = jlo; j <= jhi; ++j) *reinterpret_cast<uint4 *>(d + j * jstep) = v;
            }
    }
}

// ---------------------------------------------------------------- converter fast path

// A converter thread's column item, decoded once per kernel instead of once
// per tile.  The fast path applies when each thread owns at most one item per
// channel slab and C is a multiple of 8: it then runs a branch-free row loop.  In isolation it converts a benchmark-shaped tile in
// about half the cycles of convert_stage(), which serves every other shape.
struct ConvItem {
    bool active;        // the thread owns an item
    int px;             // image column (row tiles) or window column (strips)
    int c0;             // first channel of the item's group within a slab
    uint32_t src_col;   // bytes into a raw row at slab 0: pixel and channels (row tiles), channels only (strips)
    uint32_t dst0;      // bytes into a stage for the thread's first row rp
    uint32_t jmask;     // row tiles: the copies j that hold the pixel; strips: 1
};

template <int BITS>
__device__ __forceinline__ ConvItem conv_item(const TcArgs &a, const ConvMap &mp)
{
    ConvItem it;
    const int ncol = a.ncol_w << a.log2_groups;
    const int ci = mp.ci0;
    const int gq = ci / a.ncol_w;  // once per kernel
    const int c0 = gq * a.kch;
    it.px = ci - gq * a.ncol_w;
    it.c0 = c0;
    it.active = ci < ncol;
    if (a.strip) {
        it.src_col = static_cast<uint32_t>(c0 * BITS / 8);
        it.dst0 = static_cast<uint32_t>(gq) * a.chunk_stride + static_cast<uint32_t>(mp.rp * a.sp + it.px) * 16;
        it.jmask = 1u;
    } else {
        it.src_col = static_cast<uint32_t>(it.px * (a.c * BITS / 8) + c0 * BITS / 8);
        it.dst0 = static_cast<uint32_t>(gq) * a.chunk_stride + static_cast<uint32_t>(it.px + a.pw) * 16 +
                  static_cast<uint32_t>(mp.rp * a.ow) * 16;
        const int jlo = max(0, it.px + a.pw - a.ow + 1), jhi = min(a.kw - 1, it.px + a.pw);
        it.jmask = jhi >= jlo ? ((2u << jhi) - (1u << jlo)) : 0u;
    }
    return it;
}

// One tile of the thread's item: rows rp, rp + nph, ... < rows, kRowsPerPass
// per pass with every load issued before the stores.  The values written are
// those of convert_stage(): the staged encoding inside the image, the encoded
// zero outside it; row tiles store the copies in jmask, strips one position.
template <int BITS, int NJ, bool STRIP, bool F8>
__device__ __forceinline__ void convert_fast(const TcArgs &a, const uint8_t *raw, uint8_t *stage, const TileGeo &g,
                                             const ConvItem &it, const ConvMap &mp, int slab)
{
    // a group wholly past C keeps the encoded zero written at kernel start
    if (!it.active || slab * a.cs + it.c0 >= a.c) return;
    const uint32_t padv = F8 ? 0u : pad_half2<BITS>();
    const int nph = mp.nphase;
    const int row_bytes = static_cast<int>(a.row_bytes);
    bool col_ok = true;
    int col = static_cast<int>(it.src_col) + slab * a.cs * BITS / 8;
    if (STRIP) {
        const int ix = g.d0 - a.pw + it.px;
        col_ok = ix >= 0 && ix < a.w;
        col += ix * (a.c * BITS / 8);
    }
    const uint32_t row_out = static_cast<uint32_t>(STRIP ? a.sp : a.ow) * 16;
    const uint32_t jstep = a.copy_bytes - 16;
    // only dereferenced for rows inside the image and pixels inside a row
    const uint8_t *src = raw + (mp.rp - g.r_lo) * row_bytes + col;
    uint8_t *dst = stage + it.dst0;
    const int src_step = row_bytes * nph;
    const uint32_t dst_step = row_out * nph;
    for (int r = mp.rp; r < g.rows; r += kRowsPerPass * nph) {
        // Every load is issued: rows outside the image read the raw stage's
        // first bytes instead, and the encoded zero is selected afterwards, so
        // the loads go out back to back with no branch between them.
        uint4 v[kRowsPerPass];
#pragma unroll
        for (int u = 0; u < kRowsPerPass; ++u) {
            const int rr = r + u * nph;
            const bool ok = col_ok && rr >= g.r_lo && rr < g.r_hi;
            const uint8_t *q = ok ? src + u * src_step : raw;
            const uint4 x = F8 ? cvt_raw_f8<BITS>(q) : cvt_raw<BITS>(q);
            v[u] = ok ? x : make_uint4(padv, padv, padv, padv);
        }
#pragma unroll
        for (int u = 0; u < kRowsPerPass; ++u) {
            if (r + u * nph < g.rows) {
#pragma unroll
                for (int j = 0; j < NJ; ++j)
                    if ((it.jmask >> j) & 1u) *reinterpret_cast<uint4 *>(dst + u * dst_step + j * jstep) = v[u];
            }
        }
        src += kRowsPerPass * src_step;
        dst += kRowsPerPass * dst_step;
    }
}

template <int BITS, int LEAN>
__device__ __forceinline__ void converter_role(const TcArgs &a, uint8_t *smem, uint64_t *raw_full, uint64_t *raw_empty,
                               uint64_t *a_full, uint64_t *a_empty, volatile uint32_t *stage_info)
{
    const uint32_t stages_base = smem_addr(smem + a.off_stages);
    const bool vec = (a.c % 8) == 0;
    const ConvMap mp = conv_map(a.ncol_w << a.log2_groups);
    // encoded zero everywhere once: padding columns are never written afterwards
    {
        const uint32_t padv = a.fp8 ? 0u : pad_half2<BITS>();  // e4m3 zero is 0
        const uint4 pad4 = make_uint4(padv, padv, padv, padv);
        const uint32_t total = a.stages * a.stage_bytes / 16;
        for (uint32_t i = threadIdx.x; i < total; i += 128) sts128(stages_base + i * 16, pad4);
    }
    const ConvItem item = conv_item<BITS>(a, mp);
    int rs = 0, stage = 0;
    uint32_t r_ph = 0, a_ph = 0;
    for (int t = blockIdx.x; t < a.total_tiles; t += gridDim.x) {
        if (!warp_wait(&raw_full[rs], r_ph, a.status)) return;
        // the tile's row window and stage word, from the loader (released with raw_full)
        const int4 rec = *reinterpret_cast<const int4 *>(smem + a.off_rec + rs * 16);
        TileGeo g;
        g.rows = rec.x;
        g.r_lo = rec.y;
        g.r_hi = rec.z;
        const uint32_t info = static_cast<uint32_t>(rec.w);
        g.d0 = static_cast<int>(info & 0xFFFFu);
        const uint8_t *raw = smem + a.off_raw + rs * a.raw_bytes;
        for (int slab = 0; slab < a.nslab; ++slab) {
            if (!warp_wait(&a_empty[stage], a_ph ^ 1u, a.status)) return;
            uint8_t *st = smem + a.off_stages + stage * a.stage_bytes;
            bool staged = false;
            if constexpr (LEAN == 2) {  // row tiles, kernels at most 3 wide; e4m3 staging below INT-8
                convert_fast<BITS, 3, false, BITS != 8>(a, raw, st, g, item, mp, slab);
                staged = true;
            } else if constexpr (BITS != 8) {
                if (a.fp8) {  // always on the fast path (planner)
                    if (a.strip)
                        convert_fast<BITS, 1, true, true>(a, raw, st, g, item, mp, slab);
                    else if (a.kw <= 3)
                        convert_fast<BITS, 3, false, true>(a, raw, st, g, item, mp, slab);
                    else
                        convert_fast<BITS, 5, false, true>(a, raw, st, g, item, mp, slab);
                    staged = true;
                }
            }
            if (staged) {
            } else if (!LEAN && !a.conv_fast)  // the lean kernel runs only fast-path plans
                convert_stage<BITS>(a, raw, st, g, slab, vec, mp);
            else if (a.strip)
                convert_fast<BITS, 1, true, false>(a, raw, st, g, item, mp, slab);
            else if (a.kw <= 3)
                convert_fast<BITS, 3, false, false>(a, raw, st, g, item, mp, slab);
            else
                convert_fast<BITS, 5, false, false>(a, raw, st, g, item, mp, slab);
            if (threadIdx.x == 0) stage_info[stage] = info;  // released by this thread's arrive below
            fence_proxy_async_smem();
            mbar_arrive(&a_full[stage]);
            if (++stage == a.stages) {
                stage = 0;
                a_ph ^= 1u;
            }
        }
        mbar_arrive(&raw_empty[rs]);
        if (++rs == a.raw_stages) {
            rs = 0;
            r_ph ^= 1u;
        }
    }
}

// ---------------------------------------------------------------- bulk-copy issuers (warps 9, 10)

// Called by a whole warp; lane 0 arms `bar` with the byte count and issues the copies.
__device__ __forceinline__ void bulk_copy(uint8_t *dst, const uint8_t *src, uint32_t bytes, uint64_t *bar)
{
    if ((threadIdx.x & 31) == 0) {
        mbar_arrive_expect_tx(bar, bytes);
        for (uint32_t off = 0; off < bytes; off += kCopyChunk)
            bulk_g2s(dst + off, src + off, min(kCopyChunk, bytes - off), bar);
    }
    __syncwarp();
}

// Steps back over the last `count` armed phases of a ring and waits for each
// (their copies must land before the block exits).
__device__ __forceinline__ void drain_ring(uint64_t *full, int slot, uint32_t ph, int nslots, int count, int *status)
{
    for (int k = 0; k < nslots && k < count; ++k) {
        if (--slot < 0) {
            slot = nslots - 1;
            ph ^= 1u;
        }
        warp_wait(&full[slot], ph, status);
    }
}

// Input rows of each tile (all channels, only rows inside the image).
__device__ __forceinline__ void raw_loader_role(const TcArgs &a, uint8_t *smem, uint64_t *raw_full, uint64_t *raw_empty)
{
    int rs = 0;
    uint32_t ph = 0;
    int issued = 0;
    for (int t = blockIdx.x; t < a.total_tiles; t += gridDim.x) {
        const TileGeo g = tile_geo(a, t);
        const uint32_t info = static_cast<uint32_t>(g.d0) | (nt_run_starts(a, t) ? kInfoRunStart : 0u) |
                              (nt_run_ends(a, t) ? kInfoRunEnd : 0u);
        if (!warp_wait(&raw_empty[rs], ph ^ 1u, a.status)) break;
        // The converter takes the tile geometry from here instead of recomputing
        // it (seven reciprocal divisions on its critical path).  Lane 0 writes it
        // and then arrives on raw_full, which releases it.
        if ((threadIdx.x & 31) == 0)
            *reinterpret_cast<int4 *>(smem + a.off_rec + rs * 16) =
                make_int4(g.rows, g.r_lo, g.r_hi, static_cast<int>(info));
        const uint32_t bytes = (g.r_hi - g.r_lo) * a.row_bytes;
        if (bytes) {
            const uint8_t *src =
                a.x + (static_cast<long long>(g.img) * a.h + (g.oy_a - a.ph + g.r_lo)) * a.row_bytes;
            bulk_copy(smem + a.off_raw + rs * a.raw_bytes, src, bytes, &raw_full[rs]);
        } else if ((threadIdx.x & 31) == 0) {
            mbar_arrive(&raw_full[rs]);
        }
        ++issued;
        if (++rs == a.raw_stages) {
            rs = 0;
            ph ^= 1u;
        }
    }
    drain_ring(raw_full, rs, ph, a.raw_stages, issued, a.status);
}

// Filters: the whole set once per run of tiles with the same output-channel
// tile (resident), or one [nt x cs] tile per (slab, tap) step (streamed).
__device__ __forceinline__ void b_loader_role(const TcArgs &a, uint8_t *smem, uint64_t *b_full, uint64_t *b_empty, int nt_cols)
{
    pdl_wait();  // the filters come from the preparation kernel, which may still be running
    int bs = 0;
    uint32_t ph = 0;
    int issued = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < a.total_tiles && ok; t += gridDim.x) {
        const int nt = tile_nt(a, t);
        const uint8_t *wsrc = a.wpack + static_cast<size_t>(nt) * a.b_bytes;
        if (a.b_resident) {
            if (!nt_run_starts(a, t)) continue;
            if (!warp_wait(&b_empty[0], ph ^ 1u, a.status)) break;
            bulk_copy(smem, wsrc, a.b_bytes, &b_full[0]);
            ph ^= 1u;
            ++issued;
            continue;
        }
        for (int slab = 0; slab < a.nslab && ok; ++slab) {
            for (int tap = 0; tap < a.kh * a.kw; ++tap) {
                if (!warp_wait(&b_empty[bs], ph ^ 1u, a.status)) {
                    ok = false;
                    break;
                }
                const int kchunk = (tap * a.c_pad + slab * a.cs) / a.kch;
                bulk_copy(smem + bs * a.b_tile_bytes, wsrc + static_cast<size_t>(kchunk) * nt_cols * 16,
                          a.b_tile_bytes, &b_full[bs]);
                ++issued;
                if (++bs == a.b_stages) {
                    bs = 0;
                    ph ^= 1u;
                }
            }
        }
    }
    if (a.b_resident) drain_ring(b_full, 0, ph, 1, issued, a.status);
    else drain_ring(b_full, bs, ph, a.b_stages, issued, a.status);
}

// ---------------------------------------------------------------- MMA issuers (warps 12 and 15)

// Issues the MMAs of taps [t0, t1) of one slab: KSTEPS k-steps (16 channels each)
// per tap.  Called by the whole converged MMA warp (one elected lane issues).
// Descriptors come from uniform values only (tap offsets live in the kernel's
// parameter block), and the loop body has no conditionals, so the MMAs go out
// back to back.
template <int KSTEPS, bool F8>
__device__ __forceinline__ void issue_taps(const TcArgs &a, uint32_t d, uint64_t a_tmpl, uint64_t b_tmpl,
                                           uint32_t abase, uint32_t bbase, uint32_t tap_b16, uint32_t a_step,
                                           uint32_t b_step, int t0, int t1, uint32_t idesc)
{
#pragma unroll 4
    for (int t = t0; t < t1; ++t) {
        const uint64_t ad = a_tmpl + (abase + a.tap_a16[t]);
        const uint64_t bd = b_tmpl + (bbase + t * tap_b16);
#pragma unroll
        for (int kk = 0; kk < KSTEPS; ++kk) {
            if (F8) mma_f8_ss_warp(d, ad + kk * a_step, bd + kk * b_step, idesc, 1u);
            else mma_f16_ss_warp(d, ad + kk * a_step, bd + kk * b_step, idesc, 1u);
        }
    }
}

// MMA issue for the common case: filters resident and one channel slab per
// tile.  Each accumulator group's chunks are contiguous tap ranges issued
// back to back, with no per-segment bookkeeping between them.  The tensor
// pipe queues only a few MMAs, so any work this warp does between MMAs shows
// up as idle tensor cycles; this loop keeps that work to the waits and commits.
//
// With two issuers (one filter set for the whole kernel), issuer `sel` takes
// the CTA's tiles sel, sel + 2, ...; stage, group and their phases follow from
// the tile's position in the CTA's sequence, so one issuer's waits and commits
// overlap the other's MMAs.
template <int KSTEPS, bool F8>
__device__ __forceinline__ void mma_role_resident(const TcArgs &a, uint8_t *smem, uint32_t tmem_base,
                                                  uint64_t *a_full, uint64_t *a_empty, uint64_t *b_full,
                                                  uint64_t *b_empty, uint64_t *acc_full, uint64_t *acc_empty,
                                                  uint64_t *done, const volatile uint32_t *stage_info, uint32_t idesc,
                                                  int nt_cols, int sel, int nsel)
{
    const uint64_t a_tmpl = smem_desc(0, a.chunk_stride, a.a_sbo);
    const uint64_t b_tmpl = smem_desc(0, nt_cols * 16, 128);
    const uint32_t stages16 = smem_addr(smem + a.off_stages) >> 4;
    const uint32_t b16 = smem_addr(smem) >> 4;
    const uint32_t stage16 = a.stage_bytes >> 4;
    const uint32_t a_step = 2 * (a.chunk_stride >> 4), b_step = 2 * nt_cols;
    const uint32_t tap_b16 = (a.c_pad / a.kch) * nt_cols;
    const int chunk_taps = a.chunk_mmas / KSTEPS, taps = a.kh * a.kw;
    const int ngroups = a.ngroups, grp_chunks = a.grp_chunks, nsg = a.nsg, nchunks = a.nchunks;
    const int nstages = a.stages;
    const uint32_t grp_cols = grp_chunks * nt_cols;
    int *const status = a.status;
    // the two issuers' `done` commits both count (the barrier expects nsel arrivals)
    uint32_t b_ph = 0;
    if (nsel > 1) {  // one filter set for the whole kernel: both issuers wait for it once
        if (!warp_wait(&b_full[0], 0, status)) nsel = 0;
        tc_fence_after();
    }
    for (int i = sel, t = blockIdx.x + sel * gridDim.x; nsel > 0 && t < a.total_tiles;
         i += nsel, t += nsel * gridDim.x) {
        const int stage = i % nstages;
        if (!warp_wait(&a_full[stage], (i / nstages) & 1, status)) break;
        tc_fence_after();
        const uint32_t info = stage_info[stage];
        if (nsel == 1 && (info & kInfoRunStart)) {
            if (!warp_wait(&b_full[0], b_ph, status)) break;
            b_ph ^= 1u;
            tc_fence_after();
        }
        const uint32_t abase = stages16 + stage * stage16 + (info & a.d0_mask);
        bool ok = true;
        int t0 = 0;
        for (int sg = 0; sg < nsg; ++sg) {
            const int gc = i * nsg + sg;  // groups used so far by this CTA
            const int grp = gc % ngroups;
            if (!warp_wait(&acc_empty[grp], (gc / ngroups) & 1, status)) {
                ok = false;
                break;
            }
            tc_fence_after();
            uint32_t d = tmem_base + grp * grp_cols;
            const int last_chunk = min(nchunks, (sg + 1) * grp_chunks);
            for (int c = sg * grp_chunks; c < last_chunk; ++c) {
                const int t1 = min(t0 + chunk_taps, taps);
                issue_taps<KSTEPS, F8>(a, d, a_tmpl, b_tmpl, abase, b16, tap_b16, a_step, b_step, t0, t1, idesc);
                t0 = t1;
                d += nt_cols;
            }
            mma_commit_warp(&acc_full[grp]);
        }
        if (!ok) break;
        mma_commit_warp(&a_empty[stage]);
        if (nsel == 1 && (info & kInfoRunEnd)) mma_commit_warp(&b_empty[0]);
    }
    // every issued MMA completes before TMEM is released
    mma_commit_warp(done);
    warp_wait(done, 0, status);
}

// MMA issue, general case (streamed filters, or several channel slabs per tile).
template <bool F8>
__device__ __forceinline__ void mma_role(const TcArgs &a, uint8_t *smem, uint32_t tmem_base, uint64_t *a_full,
                                         uint64_t *a_empty, uint64_t *b_full, uint64_t *b_empty, uint64_t *acc_full,
                                         uint64_t *acc_empty, uint64_t *done, const volatile uint32_t *stage_info,
                                         uint32_t idesc, int nt_cols)
{
    const uint32_t b_lbo = nt_cols * 16;
    const uint64_t a_tmpl = smem_desc(0, a.chunk_stride, a.a_sbo);
    const uint64_t b_tmpl = smem_desc(0, b_lbo, 128);
    const uint32_t stages16 = smem_addr(smem + a.off_stages) >> 4;
    const uint32_t b16 = smem_addr(smem) >> 4;
    const uint32_t stage16 = a.stage_bytes >> 4, btile16 = a.b_tile_bytes >> 4;
    const uint32_t a_step = 2 * (a.chunk_stride >> 4), b_step = 2 * nt_cols;  // one k-step = two K-chunks
    const uint32_t slab_b16 = (a.cs / a.kch) * nt_cols;
    const int ksteps = a.cs / (2 * a.kch);
    const bool resident = a.b_resident != 0;
    // resident filters: tap t of slab s sits at t * c_pad/kch chunks; streamed: each tap has its own tile
    const uint32_t tap_b16 = resident ? (a.c_pad / a.kch) * nt_cols : 0;
    const int chunk_taps = a.chunk_mmas / ksteps, taps = a.kh * a.kw;
    const int nslab = a.nslab, nstages = a.stages, nbstages = a.b_stages;
    const int grp_chunks = a.grp_chunks, ngroups = a.ngroups, nchunks = a.nchunks;
    int *const status = a.status;
    int stage = 0, bs = 0, grp = 0;
    uint32_t a_ph = 0, b_ph = 0, empty_ph = 0;
    bool ok = true;
    // The tile sequence matches the converter's; the tile's pixel offset and
    // filter-run flags come with each stage (no per-tile geometry here).
    for (int t = blockIdx.x; t < a.total_tiles && ok; t += gridDim.x) {
        int in_chunk = 0, chunk = 0, sub = 0;  // MMAs into the current chunk, chunk of the tile, buffer in the group
        uint32_t info = 0;
        for (int slab = 0; slab < nslab && ok; ++slab) {
            if (!warp_wait(&a_full[stage], a_ph, status)) {
                ok = false;
                break;
            }
            tc_fence_after();
            info = stage_info[stage];
            if (slab == 0 && resident && (info & kInfoRunStart)) {
                if (!warp_wait(&b_full[0], b_ph, status)) {
                    ok = false;
                    break;
                }
                b_ph ^= 1u;
                tc_fence_after();
            }
            const uint32_t abase = stages16 + stage * stage16 + (info & a.d0_mask);
            int tap = 0;
            while (tap < taps) {
                uint32_t bbase = b16 + slab * slab_b16;
                int seg = taps - tap;
                if (!resident) {  // one streamed filter tile per tap
                    if (!warp_wait(&b_full[bs], b_ph, status)) {
                        ok = false;
                        break;
                    }
                    bbase = b16 + bs * btile16 - tap * tap_b16;
                    seg = 1;
                }
                if (in_chunk == 0 && sub == 0) {  // a new accumulator group
                    if (!warp_wait(&acc_empty[grp], (empty_ph >> grp) & 1u, status)) {
                        ok = false;
                        break;
                    }
                    empty_ph ^= 1u << grp;
                    tc_fence_after();
                }
                seg = min(seg, chunk_taps - in_chunk);
                const uint32_t d = tmem_base + (grp * grp_chunks + sub) * nt_cols;
                if (ksteps == 1)
                    issue_taps<1, F8>(a, d, a_tmpl, b_tmpl, abase, bbase, tap_b16, a_step, b_step, tap, tap + seg, idesc);
                else if (ksteps == 2)
                    issue_taps<2, F8>(a, d, a_tmpl, b_tmpl, abase, bbase, tap_b16, a_step, b_step, tap, tap + seg, idesc);
                else
                    issue_taps<4, F8>(a, d, a_tmpl, b_tmpl, abase, bbase, tap_b16, a_step, b_step, tap, tap + seg, idesc);
                tap += seg;
                in_chunk += seg;
                if (in_chunk == chunk_taps || (slab == nslab - 1 && tap == taps)) {  // chunk complete
                    in_chunk = 0;
                    ++chunk;
                    if (++sub == grp_chunks || chunk == nchunks) {  // group complete
                        mma_commit_warp(&acc_full[grp]);
                        sub = 0;
                        if (++grp == ngroups) grp = 0;
                    }
                }
                if (!resident) {
                    mma_commit_warp(&b_empty[bs]);
                    if (++bs == nbstages) {
                        bs = 0;
                        b_ph ^= 1u;
                    }
                }
            }
            if (!ok) break;
            mma_commit_warp(&a_empty[stage]);
            if (++stage == nstages) {
                stage = 0;
                a_ph ^= 1u;
            }
        }
        if (ok && resident && (info & kInfoRunEnd)) mma_commit_warp(&b_empty[0]);
    }
    // every issued MMA completes before TMEM is released
    mma_commit_warp(done);
    warp_wait(done, 0, status);
}

// ---------------------------------------------------------------- epilogue (warps 4-11)

// TMEM access in steps of 16 (or, for 8-column warps, 8) columns.
template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t (&v)[N])
{
    if (N == 8) {
        uint32_t t[8];
        tmem_ld8(taddr, t);
#pragma unroll
        for (int k = 0; k < 8; ++k) v[k] = t[k];
    } else {
#pragma unroll
        for (int c = 0; c < N; c += 16) {
            uint32_t t[16];
            tmem_ld16(taddr + c, t);
#pragma unroll
            for (int k = 0; k < 16; ++k) v[c + k] = t[k];
        }
    }
}

template <int N>
__device__ __forceinline__ void tmem_st_cols(uint32_t taddr, const uint32_t (&v)[N])
{
    if (N == 8) {
        uint32_t t[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) t[k] = v[k];
        tmem_st8(taddr, t);
    } else {
#pragma unroll
        for (int c = 0; c < N; c += 16) {
            uint32_t t[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) t[k] = v[c + k];
            tmem_st16(taddr + c, t);
        }
    }
}

template <int N>
__device__ __forceinline__ void tmem_fill_cols(uint32_t taddr, uint32_t value)
{
    if (N == 8) {
        tmem_st8_fill(taddr, value);
    } else {
#pragma unroll
        for (int c = 0; c < N; c += 16) tmem_st16_fill(taddr + c, value);
    }
}

// Barrier among the epilogue warps only (named barrier 1).
__device__ __forceinline__ void epi_barrier()
{
    asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
}

// Releases an accumulator buffer: this warp's TMEM stores are complete before
// one lane arrives (the barrier counts one arrival per epilogue warp).
__device__ __forceinline__ void release_acc(uint64_t *bar)
{
    tmem_wait_st();
    tc_fence_before();
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}

// Epilogue warps: warp w reads TMEM lane quarter w % 4 (tile rows = output
// pixels) and one half of the NT columns.  Per accumulator group it adds the
// group's buffers (the raw fp32 bit patterns, an exact integer sum, see the
// prep kernel) in batches of up to 32 columns, puts the accumulator pre-load
// back and releases the group before the compression arithmetic, so the MMA
// warp can refill it meanwhile.  Tiles that take several groups carry their
// running sums in TMEM.
template <int BITS, int NT, bool POOL, int LEAN>
__device__ __forceinline__ void epilogue_role(const TcArgs &a, uint8_t *smem, uint32_t tmem_base, uint64_t *acc_full,
                                              uint64_t *acc_empty)
{
    constexpr int CW = NT / 2;                  // columns of this warp
    constexpr int BATCH = CW < 16 ? CW : 16;   // columns per TMEM wait
    constexpr int G = CW < 16 ? CW : 16;       // channels per compression group
    constexpr int kMaxSrc = 512 / NT / 2 + 1;  // buffers of one group (planner bound) plus the running sums
    const int warp = threadIdx.x >> 5;
    const int quarter = warp & 3;
    const int half = (warp - kConvWarps) >> 2;
    const int lane = threadIdx.x & 31;
    const int row = quarter * 32 + lane;  // tile row = output pixel within the tile
    const int col0 = half * CW;
    const int grp_chunks = a.grp_chunks, ngroups = a.ngroups, nsg = a.nsg, nchunks = a.nchunks;
    const uint32_t lane_addr = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + col0;
    const uint32_t sum_addr = lane_addr + ngroups * grp_chunks * NT;
    const int mp = a.n_ntiles * NT;
    const int4 *rec0 = reinterpret_cast<const int4 *>(smem + a.off_chan);
    const int4 *rec1 = rec0 + mp;
    const uint8_t *gdirect = reinterpret_cast<const uint8_t *>(rec1 + mp);  // per 16-channel group
    const int pix_per_img = a.oh * a.ow;
    const int out_row_bytes = a.m * BITS / 8;
    const int m = a.m;
    uint8_t *const ybase = a.y;
    int *const status = a.status;

    for (int b = 0; b < ngroups * grp_chunks; ++b) tmem_fill_cols<CW>(lane_addr + b * NT, kMagic);
    tmem_wait_st();
    tc_fence_before();
    __syncwarp();
    if (lane == 0)
        for (int b = 0; b < ngroups; ++b) mbar_arrive(&acc_empty[b]);
    // compression records (written by the preparation kernel, which may still be
    // running), plus one "all direct" flag per 16-channel group
    pdl_wait();
    {
        int4 *chan = reinterpret_cast<int4 *>(smem + a.off_chan);
        const int et = threadIdx.x - kConvWarps * 32, ne = kEpiWarps * 32;
        for (int i = et; i < 2 * mp; i += ne) {
            int4 r = a.chan[i];
            if (i < mp && r.w == kModeThreshold) r.x = static_cast<int>(a.off_thr) + i * 4 * kThrStride;
            chan[i] = r;
        }
        uint8_t *gd = reinterpret_cast<uint8_t *>(chan + 2 * mp);
        for (int gi = et; gi < mp / 16; gi += ne) {
            int all = 1;
            for (int k = 0; k < 16; ++k) all &= a.chan[gi * 16 + k].w == kModeDirect;
            gd[gi] = static_cast<uint8_t>(all);
        }
        if (a.thr) {
            int32_t *ts = reinterpret_cast<int32_t *>(smem + a.off_thr);
            for (int i = et; i < mp * kThrStride; i += ne) ts[i] = a.thr[i];
        }
        epi_barrier();
    }

    uint32_t full_ph = 0;
    int grp = 0;
    for (int t = blockIdx.x; t < a.total_tiles; t += gridDim.x) {
        const TileGeo g = tile_geo(a, t);
        // Pixels past the end of the image are computed but not stored.  TMEM
        // accesses are warp-collective, so every lane executes them; only the
        // store depends on the lane's pixel.
        int p;
        bool pix_ok;
        if (a.strip) {  // tile row = 8 * (output row - oy_a) + (output column - d0)
            const int oy = g.oy_a + (row >> 3), ox = g.d0 + (row & 7);
            pix_ok = oy < a.oh && ox < a.ow;
            p = oy * a.ow + ox;
        } else {
            p = g.ti * kTileM + row;
            pix_ok = p < pix_per_img;
        }
        const int m0 = g.nt * NT + col0;
        uint8_t *dst_row =
            ybase + (static_cast<long long>(g.img) * pix_per_img + (pix_ok ? p : 0)) * out_row_bytes;
        // Fused 2x2/2 max-pool (strip tiles): the window of pooled pixel
        // (oy/2, ox/2) is tile rows 8*dy + dx apart, lanes L, L^1, L^8, L^9 of
        // one warp; its top-left lane stores.  Windows that reach past the
        // image have no pooled pixel (floor output size).
        bool pool_store = false;
        uint8_t *pool_row = ybase;
        if constexpr (POOL) {
            const int oy = g.oy_a + (row >> 3), ox = g.d0 + (row & 7);
            pool_store = (row & 9) == 0 && (oy >> 1) < a.pool_oh && (ox >> 1) < a.pool_ow;
            if (pool_store)
                pool_row += ((static_cast<long long>(g.img) * a.pool_oh + (oy >> 1)) * a.pool_ow + (ox >> 1)) * out_row_bytes;
        }
        for (int sg = 0; sg < nsg; ++sg) {
            if (!warp_wait(&acc_full[grp], (full_ph >> grp) & 1u, status)) return;
            full_ph ^= 1u << grp;
            tc_fence_after();
            const int nsub = min(grp_chunks, nchunks - sg * grp_chunks);
            const uint32_t grp_addr = lane_addr + grp * grp_chunks * NT;
            const bool last = sg == nsg - 1;
            uint32_t v[CW];
            bool drained = false;
            if constexpr (CW == 32) {
                if (nsg == 1 && nsub <= 2) {
                    // the whole tile in one group of one or two buffers: per
                    // half of the warp's columns, every load in flight, one wait
#pragma unroll
                    for (int b0 = 0; b0 < 32; b0 += 16) {
                        uint32_t t0[16], t1[16];
                        tmem_ld16(grp_addr + b0, t0);
                        if (nsub == 2) tmem_ld16(grp_addr + NT + b0, t1);
                        tmem_wait_ld();
#pragma unroll
                        for (int k = 0; k < 16; ++k) v[b0 + k] = nsub == 2 ? t0[k] + t1[k] : t0[k];
                        tmem_st16_fill(grp_addr + b0, kMagic);
                        if (nsub == 2) tmem_st16_fill(grp_addr + NT + b0, kMagic);
                    }
                    drained = true;
                }
            }
            if (!LEAN && !drained) {  // the lean kernel runs only one-group, at most two-buffer plans
#pragma unroll
            for (int k = 0; k < CW; ++k) v[k] = 0;
            const int nsrc = nsub + (sg > 0 ? 1 : 0);
#pragma unroll
            for (int sub = 0; sub < kMaxSrc; ++sub) {  // unrolled: v[] stays in registers
                // the group's buffers, then (for a tile's later groups) its running sums
                if (sub >= nsrc) break;
                const bool is_sum = sub == nsub;
                const uint32_t src = is_sum ? sum_addr : grp_addr + sub * NT;
#pragma unroll
                for (int b0 = 0; b0 < CW; b0 += BATCH) {
                    uint32_t tmp[BATCH];
                    tmem_ld_cols<BATCH>(src + b0, tmp);
                    tmem_wait_ld();
#pragma unroll
                    for (int k = 0; k < BATCH; ++k) v[b0 + k] += tmp[k];
                    if (!is_sum) tmem_fill_cols<BATCH>(src + b0, kMagic);
                }
            }
            }
            if (!last) {
#pragma unroll
                for (int b0 = 0; b0 < CW; b0 += BATCH) {
                    uint32_t tmp[BATCH];
#pragma unroll
                    for (int k = 0; k < BATCH; ++k) tmp[k] = v[b0 + k];
                    tmem_st_cols<BATCH>(sum_addr + b0, tmp);
                }
            }
            release_acc(&acc_empty[grp]);
            if (++grp == ngroups) grp = 0;
            if (POOL && last) {
#pragma unroll
                for (int c = 0; c < CW; c += G) {
                    const int valid = m - (m0 + c);  // same for the whole warp: every lane shuffles
                    if (valid > 0) {
                        uint32_t pk[(G * BITS + 31) / 32];
                        compress_pack<BITS, G>(v + c, rec0, rec1, gdirect[(m0 + c) >> 4] != 0, m0 + c, pk);
#pragma unroll
                        for (int wd = 0; wd < (G * BITS + 31) / 32; ++wd) {
                            pk[wd] = max_fields<BITS>(pk[wd], __shfl_xor_sync(0xffffffffu, pk[wd], 1));
                            pk[wd] = max_fields<BITS>(pk[wd], __shfl_xor_sync(0xffffffffu, pk[wd], 8));
                        }
                        if (pool_store) store_packed<BITS, G>(pk, valid, pool_row + (m0 + c) * BITS / 8);
                    }
                }
            } else if (last && pix_ok) {
#pragma unroll
                for (int c = 0; c < CW; c += G) {
                    const int valid = m - (m0 + c);  // same for the whole warp
                    if (valid > 0)
                        compress_store<BITS, G>(v + c, rec0, rec1, gdirect[(m0 + c) >> 4] != 0, m0 + c, valid,
                                                dst_row + (m0 + c) * BITS / 8);
                }
            }
        }
    }
}

// POOL: the fused 2x2/2 max-pool epilogue (a separate instantiation, so the
// plain kernel carries none of its registers).
// LEAN 1: only the hot paths of the common plans (converter fast path,
// resident filters in one slab, one accumulator group of at most two buffers,
// NT = 64).  LEAN 2: of those, only row tiles of kernels at most 3 wide with
// 32 channels per tap: fp16 staging and two k-steps per tap at INT-8, e4m3
// staging and one k-step per tap at INT-4/INT-2.  Each SM
// sub-partition runs four warps of different roles from this one kernel, and
// code for other plans stalls their instruction fetch.
template <int BITS, int NT, bool POOL, int LEAN>
__global__ void __launch_bounds__(kThreads, 1) conv_tc_kernel(const TcArgs a)
{
    extern __shared__ __align__(128) uint8_t smem[];
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + a.off_bar);
    uint64_t *raw_full = bars;
    uint64_t *raw_empty = raw_full + a.raw_stages;
    uint64_t *a_full = raw_empty + a.raw_stages;
    uint64_t *a_empty = a_full + a.stages;
    uint64_t *b_full = a_empty + a.stages;
    uint64_t *b_empty = b_full + a.b_stages;
    uint64_t *acc_full = b_empty + a.b_stages;
    uint64_t *acc_empty = acc_full + kMaxAccGroups;
    uint64_t *done = acc_empty + kMaxAccGroups;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
    volatile uint32_t *stage_info = tmem_slot + 1;  // kMaxStages words
    const int warp = threadIdx.x >> 5;

    if (warp == kMmaWarp) {
        if ((threadIdx.x & 31) == 0) {
            for (int s = 0; s < a.raw_stages; ++s) {
                mbar_init(&raw_full[s], 1);
                mbar_init(&raw_empty[s], 128);
            }
            for (int s = 0; s < a.stages; ++s) {
                mbar_init(&a_full[s], 128);
                mbar_init(&a_empty[s], 1);
            }
            for (int s = 0; s < a.b_stages; ++s) {
                mbar_init(&b_full[s], 1);
                mbar_init(&b_empty[s], 1);
            }
            for (int b = 0; b < kMaxAccGroups; ++b) {
                mbar_init(&acc_full[b], 1);
                mbar_init(&acc_empty[b], kEpiWarps);
            }
            mbar_init(done, a.mma_warps);
            fence_mbar_init();
        }
        __syncwarp();
        tmem_alloc(tmem_slot, a.tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp < kConvWarps) {
        converter_role<BITS, LEAN>(a, smem, raw_full, raw_empty, a_full, a_empty, stage_info);
    } else if (warp < kConvWarps + kEpiWarps) {
        epilogue_role<BITS, NT, POOL, LEAN>(a, smem, tmem_base, acc_full, acc_empty);
    } else if (warp == kMmaWarp || (warp == kMmaWarp2 && a.mma_warps == 2)) {
        // the instruction descriptor is the same for both kinds (format fields 0: f16 / e4m3)
        const uint32_t idesc = idesc_f16_f32(kTileM, NT);
        const int sel = warp == kMmaWarp ? 0 : 1;
        const int ks = a.cs / (2 * a.kch);  // k-steps per tap and slab
        bool issued = false;
        if constexpr (LEAN == 2) {
            mma_role_resident<BITS == 8 ? 2 : 1, BITS != 8>(a, smem, tmem_base, a_full, a_empty, b_full, b_empty,
                                                            acc_full, acc_empty, done, stage_info, idesc, NT, sel,
                                                            a.mma_warps);
            issued = true;
        } else if constexpr (BITS != 8) {
            if (a.fp8) {
                if (a.b_resident && a.nslab == 1 && ks == 1)
                    mma_role_resident<1, true>(a, smem, tmem_base, a_full, a_empty, b_full, b_empty, acc_full,
                                               acc_empty, done, stage_info, idesc, NT, sel, a.mma_warps);
                else if (a.b_resident && a.nslab == 1 && ks == 2)
                    mma_role_resident<2, true>(a, smem, tmem_base, a_full, a_empty, b_full, b_empty, acc_full,
                                               acc_empty, done, stage_info, idesc, NT, sel, a.mma_warps);
                else if (!LEAN)
                    mma_role<true>(a, smem, tmem_base, a_full, a_empty, b_full, b_empty, acc_full, acc_empty, done,
                                   stage_info, idesc, NT);
                issued = true;
            }
        }
        if (issued) {
        } else if (a.b_resident && a.nslab == 1 && ks == 2)
            mma_role_resident<2, false>(a, smem, tmem_base, a_full, a_empty, b_full, b_empty, acc_full, acc_empty, done,
                                        stage_info, idesc, NT, sel, a.mma_warps);
        else if (a.b_resident && a.nslab == 1 && ks == 4)
            mma_role_resident<4, false>(a, smem, tmem_base, a_full, a_empty, b_full, b_empty, acc_full, acc_empty, done,
                                        stage_info, idesc, NT, sel, a.mma_warps);
        else if (a.b_resident && a.nslab == 1)
            mma_role_resident<1, false>(a, smem, tmem_base, a_full, a_empty, b_full, b_empty, acc_full, acc_empty, done,
                                        stage_info, idesc, NT, sel, a.mma_warps);
        else if (!LEAN)
            mma_role<false>(a, smem, tmem_base, a_full, a_empty, b_full, b_empty, acc_full, acc_empty, done, stage_info,
                            idesc, NT);
    } else if (warp == kRawWarp) {
        raw_loader_role(a, smem, raw_full, raw_empty);
    } else if (warp == kBWarp) {
        b_loader_role(a, smem, b_full, b_empty, NT);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, a.tmem_cols);
    }
}

// ---------------------------------------------------------------- filter / constant preparation

// One warp per (padded) output channel: fp16 filters in the [ntile][k/8][nt][8]
// layout of the B operand, and the channel's compression records:
//   rec0 = {lam2, kappa, shift, mode}, rec1 = {beta, ulo, uhi, lambda}
// where the epilogue's raw sum s (sum of the chunks' bit patterns) relates to the
// accumulator by acc + bias = s + beta (mod 2^32), and lam2 = beta*kappa + lambda
// (mod 2^32).  Mode "direct" holds when (acc + bias)*kappa + lambda fits int32 for
// every accumulator this channel's weights can produce (activations in
// [0, 2^Q-1]); mode "clamp" when the saturation bounds allow a 32-bit form.
// The kernel lets the convolution that follows it start at once (that kernel
// waits for these results only where it reads them).
template <int BITS>
__global__ void __launch_bounds__(256) conv_tc_prep_kernel(const uint8_t *w, const int32_t *bias, const int16_t *kappa,
                                                           const int32_t *lambda, const uint8_t *shifts, int shift,
                                                           int m, int mp, int kh, int kw, int c, int c_pad, int k_pad,
                                                           int nt, int nchunks, int fp8, uint16_t *wpack, int4 *chan,
                                                           const int32_t *thresholds, int32_t *thr_out)
{
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const int o = blockIdx.x * 8 + (threadIdx.x >> 5);
    if (o >= mp) return;
    const int tile = o / nt, col = o - tile * nt;
    const int taps = kh * kw;
    const int slot_of[8] = {0, 2, 4, 6, 1, 3, 5, 7};  // inverse of {0,4,1,5,2,6,3,7}
    int sum = 0, pos = 0, neg = 0;  // |sum| <= K * 2^(Q-1) < 2^31 (accumulator bound of the ABI)
    for (int tap = 0; tap < taps; ++tap) {
        for (int cc = lane; cc < c_pad; cc += 32) {  // consecutive lanes: consecutive channels and slots
            int v = 0;
            if (o < m && cc < c) {
                const long long e = (static_cast<long long>(o) * taps + tap) * c + cc;
                if (BITS == 8) {
                    v = static_cast<int8_t>(w[e]);
                } else {
                    constexpr int per = 8 / BITS;
                    const int f = (w[e / per] >> ((e % per) * BITS)) & ((1 << BITS) - 1);
                    v = f >= (1 << (BITS - 1)) ? f - (1 << BITS) : f;
                }
            }
            sum += v;
            pos += max(v, 0);
            neg += min(v, 0);
            const int k = tap * c_pad + cc;
            if (fp8) {
                // e4m3 bytes, 16 channels per K-chunk; INT-2 in the converter's word order
                const int ch = cc & 15;
                const int slot = BITS == 4 ? ch : (ch & 8) + (ch & 1) * 4 + ((ch & 7) >> 1);
                const size_t dst = ((static_cast<size_t>(tile) * (k_pad / 16) + k / 16) * nt + col) * 16 + slot;
                reinterpret_cast<uint8_t *>(wpack)[dst] = e4m3_of_int(v);
            } else {
                const int slot = BITS == 8 ? (cc & 7) : slot_of[cc & 7];
                const size_t dst = ((static_cast<size_t>(tile) * (k_pad / 8) + k / 8) * nt + col) * 8 + slot;
                wpack[dst] = __half_as_ushort(__int2half_rn(v));
            }
        }
    }
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
        sum += __shfl_xor_sync(0xffffffffu, sum, d);
        pos += __shfl_xor_sync(0xffffffffu, pos, d);
        neg += __shfl_xor_sync(0xffffffffu, neg, d);
    }
    if (thresholds) {  // staircase compression: the channel's thresholds, padded channels never step up
        for (int k = lane; k < kThrStride; k += 32)
            thr_out[o * kThrStride + k] =
                (o < m && k < (1 << BITS) - 1) ? thresholds[static_cast<long long>(o) * ((1 << BITS) - 1) + k] : INT32_MAX;
    }
    if (lane == 0 && thresholds) {
        // the epilogue compares acc = s + beta (bias is part of the thresholds)
        const long long off = fp8 ? 0 : (BITS == 8) ? -128 : 1024;
        const uint32_t beta = 0u - static_cast<uint32_t>(off * sum) - static_cast<uint32_t>(nchunks) * kMagic;
        chan[o] = make_int4(0, 0, 0, kModeThreshold);  // .x: threshold location, set when staged
        chan[mp + o] = make_int4(static_cast<int32_t>(beta), 0, 0, 0);
    } else if (lane == 0) {
        int4 r0 = make_int4(0, 0, 0, kModeDirect), r1 = make_int4(0, 0, 0, 0);
        if (o < m) {
            const long long off = fp8 ? 0 : (BITS == 8) ? -128 : 1024;  // staged activation = x + off
            const int32_t b = bias ? bias[o] : 0;
            const uint32_t beta = static_cast<uint32_t>(b) - static_cast<uint32_t>(off * sum) -
                                  static_cast<uint32_t>(nchunks) * kMagic;
            const int32_t kap = kappa[o], lam = lambda[o], sh = shifts ? shifts[o] : shift;
            const long long top = (1 << BITS) - 1;
            // every accumulator of this channel lies in [top * neg, top * pos]
            const long long u0 = top * neg + b, u1 = top * pos + b;
            const bool direct = in_i32(u0 * kap + lam) && in_i32(u1 * kap + lam);
            long long ulo = 0, uhi = 0;
            const bool clamp = !direct && saturation_bounds(kap, lam, sh, top, &ulo, &uhi);
            const int mode = direct ? kModeDirect : clamp ? kModeClamp : kModeWide;
            const uint32_t lam2 = beta * static_cast<uint32_t>(kap) + static_cast<uint32_t>(lam);
            r0 = make_int4(static_cast<int32_t>(lam2), kap, sh, mode);
            r1 = make_int4(static_cast<int32_t>(beta), static_cast<int32_t>(ulo), static_cast<int32_t>(uhi), lam);
        }
        chan[o] = r0;
        chan[mp + o] = r1;
    }
}

template <int BITS, int NT, bool POOL, int LEAN = 0>
cudaError_t launch_tc(const TcArgs &args, int grid, uint32_t smem, cudaStream_t st, bool after_prep)
{
    // the opt-in shared-memory limit is raised once per device, outside any stream capture
    static std::mutex mu;
    static bool raised[64] = {};
    auto kern = conv_tc_kernel<BITS, NT, POOL, LEAN>;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
        if (!raised[dev]) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
            if (e != cudaSuccess) return e;
            raised[dev] = true;
        }
    }
    if (!after_prep) {
        kern<<<grid, kThreads, smem, st>>>(args);
        return cudaGetLastError();
    }
    // Right after the preparation kernel: start while it still runs.  Only the
    // filter loader and the epilogue's record load wait for its results.
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, args);
}

template <int BITS>
cudaError_t launch_tc_bits(int nt, const TcArgs &args, int grid, uint32_t smem, cudaStream_t st, bool after_prep)
{
    switch (nt) {
        case 16: return args.pool ? launch_tc<BITS, 16, true>(args, grid, smem, st, after_prep)
                                  : launch_tc<BITS, 16, false>(args, grid, smem, st, after_prep);
        case 32: return args.pool ? launch_tc<BITS, 32, true>(args, grid, smem, st, after_prep)
                                  : launch_tc<BITS, 32, false>(args, grid, smem, st, after_prep);
        case 64: {
            // the lean kernel serves plans whose every path it compiles (see conv_tc_kernel)
            const bool lean = args.conv_fast && args.b_resident && args.nslab == 1 && args.nsg == 1 && args.nchunks <= 2;
            // INT-8 with fp16 staging, or INT-4/INT-2 with e4m3 staging, at 32 channels per tap
            if (lean && !args.pool && !args.strip && args.kw <= 3 && args.cs == 32 && (BITS == 8) == !args.fp8)
                return launch_tc<BITS, 64, false, 2>(args, grid, smem, st, after_prep);
            if (lean)
                return args.pool ? launch_tc<BITS, 64, true, 1>(args, grid, smem, st, after_prep)
                                 : launch_tc<BITS, 64, false, 1>(args, grid, smem, st, after_prep);
            return args.pool ? launch_tc<BITS, 64, true>(args, grid, smem, st, after_prep)
                             : launch_tc<BITS, 64, false>(args, grid, smem, st, after_prep);
        }
        case 128: return args.pool ? launch_tc<BITS, 128, true>(args, grid, smem, st, after_prep)
                                   : launch_tc<BITS, 128, false>(args, grid, smem, st, after_prep);
        default: return cudaErrorInvalidValue;
    }
}

uint32_t round_up(uint32_t v, uint32_t a) { return (v + a - 1) / a * a; }

size_t chan_offset(const TcPlan &plan)
{
    return (static_cast<size_t>(plan.n_ntiles) * plan.b_bytes + 255) / 256 * 256;
}

}  // namespace

namespace {

// One layout: fp16 staging (K = 16 channels per MMA), or for INT-4/INT-2 with
// C a multiple of 32, e4m3 staging (K = 32).  The e4m3 embedding is exact: the
// values lie in [-8, 15], each e4m3 product is an integer up to 15 * 8, and a
// probe of the kind::f8f6f4 MMA against int64 sums (K up to 1024, adversarial
// orderings, with and without the accumulator pre-load) found no error.
TcPlan plan_layout(const ConvShape &s, bool fp8)
{
    TcPlan p{};
    p.ok = false;
    p.fp8 = fp8;
    const int kch = fp8 ? 16 : 8;  // channels per 16-byte K-chunk
    const uint32_t eb = fp8 ? 1 : 2;  // bytes per staged element
    if (s.sh != 1 || s.sw != 1 || s.oh <= 0 || s.ow <= 0) return p;
    if (s.kh * s.kw > kMaxTaps || s.kw > 32) return p;  // per-tap table; 32-bit copy mask
    const long long row_bytes = static_cast<long long>(s.w) * s.c * s.bits / 8;
    if (row_bytes % 16 != 0 || row_bytes > (1 << 20)) return p;  // rows move as whole bulk copies
    const int mp16 = (s.m + 15) / 16 * 16;
    p.nt = mp16 <= 16 ? 16 : mp16 <= 32 ? 32 : mp16 <= 64 ? 64 : 128;
    p.n_ntiles = (s.m + p.nt - 1) / p.nt;
    p.c_pad = (s.c + 2 * kch - 1) / (2 * kch) * (2 * kch);
    p.k_pad = s.kh * s.kw * p.c_pad;
    p.row_bytes = static_cast<uint32_t>(row_bytes);
    // A tile's 128 MMA rows are 16 groups of 8 consecutive output pixels of one
    // row, and the A descriptor steps between groups by one fixed stride.  Row
    // tiles take 128 consecutive pixels (groups 128 B apart) and need kw copies
    // of the staged rows, copy j shifted by j pixels, because a tap's column
    // shift wraps around the row ends.  Strip tiles take 16 output rows by 8
    // columns: group g is output row oy_a + g, the stride is the staged window
    // width, and every tap (i, j) is the offset i * sp + j into a single padded
    // window of (16 + kh - 1) x (8 + kw - 1) pixels.  Strips need kw times fewer
    // converter stores; they are chosen unless their count (partial strips at
    // the right and bottom edges compute pixels that are not stored) exceeds
    // that of row tiles by more than 15 %, or row tiles cover whole output rows
    // of a kernel at most 3 wide exactly (ow divides 128, images hold whole
    // tiles): there row tiles stage only the rows they need and measure ~3 %
    // faster (3x3, 16x16 images), while strips load full input rows.
    const long long rm_tiles = (static_cast<long long>(s.oh) * s.ow + kTileM - 1) / kTileM;
    p.ncb = (s.ow + kStripCols - 1) / kStripCols;
    const long long strip_tiles = static_cast<long long>(p.ncb) * ((s.oh + kStripRows - 1) / kStripRows);
    const bool rows_exact = s.kw <= 3 && s.ow >= 16 && kTileM % s.ow == 0 && (s.oh * s.ow) % kTileM == 0;
    p.strip = s.kw > 1 && s.ow < 16384 && !rows_exact && strip_tiles * 100 <= rm_tiles * 115;
    if (s.pool) {  // the fused pool needs each 2x2 window inside one warp: strips only
        if (s.ow >= 16384) return p;
        p.strip = true;
    }
    if (p.strip) {
        p.sp = kStripCols + s.kw - 1;
        p.rows_max = std::min(kStripRows, s.oh) + s.kh - 1;
        // the MMA addresses all 16 groups' rows, stored or not
        p.p_alloc = static_cast<int>(round_up(static_cast<uint32_t>((kStripRows + s.kh - 1) * p.sp), 8));
    } else {
        p.sp = 0;
        const int out_rows = std::min((s.ow - 1 + kTileM + s.ow - 1) / s.ow, s.oh);
        p.rows_max = out_rows + s.kh - 1;
        // positions per copy: the staged rows, and at least everything the 128 tile rows can address
        const int reach = (s.ow - 1) + kTileM + (s.kh - 1) * s.ow;
        p.p_alloc = static_cast<int>(round_up(static_cast<uint32_t>(std::max(p.rows_max * s.ow, reach)), 8));
    }
    if (p.p_alloc * 16 >= (1 << 18)) return p;  // descriptor offset field
    p.raw_bytes = round_up(static_cast<uint32_t>(p.rows_max * row_bytes), 128);
    if (p.raw_bytes >= (1u << 20)) return p;    // single transaction count
    p.b_bytes = static_cast<uint32_t>(p.nt) * p.k_pad * eb;
    p.mmas_per_tile = p.k_pad / (2 * kch);
    // products per exact chunk: |staged x| * |w| <= 2^14 (INT-8), 1039*8 (INT-4), 1027*2 (INT-2);
    // e4m3 staging has no offset: 15*8 (INT-4), 3*2 (INT-2)
    const long long max_prod = fp8 ? (s.bits == 4 ? 15 * 8 : 3 * 2)
                                   : s.bits == 8 ? 16384 : s.bits == 4 ? 1039 * 8 : 1027 * 2;
    const int limit = static_cast<int>(((1ll << 22) / max_prod) / (2 * kch));  // MMAs per exact chunk
    p.limit_mmas = limit;
    const int mp = p.n_ntiles * p.nt;
    const uint32_t thr_bytes = s.thr ? static_cast<uint32_t>(mp) * 4 * kThrStride : 0;
    const uint32_t chan_bytes = round_up(mp * 32 + mp / 16, 16) + thr_bytes;
    p.raw_stages = 2;
    for (int resident = 1; resident >= 0 && !p.cs; --resident) {
        if (resident && p.b_bytes > 120u * 1024u) continue;
        for (int cs : {64, 32, 16}) {
            if (cs > p.c_pad || p.c_pad % cs || cs < 2 * kch) continue;
            for (int stages : {3, 2}) {
                for (int bst : {4, 3, 2}) {
                    if (resident && bst != 4) continue;
                    const int b_stages = resident ? 1 : bst;
                    const uint32_t b_tile = static_cast<uint32_t>(p.nt) * cs * eb;
                    const uint32_t b_region = resident ? round_up(p.b_bytes, 128) : b_stages * b_tile;
                    const uint32_t copy_bytes = static_cast<uint32_t>(p.p_alloc) * cs * eb;
                    const uint32_t stage_bytes = copy_bytes * (p.strip ? 1 : s.kw);
                    const uint32_t off_raw = round_up(b_region, 128);
                    const uint32_t off_stages = off_raw + p.raw_stages * p.raw_bytes;
                    const uint32_t off_chan = off_stages + stages * stage_bytes;
                    const uint32_t off_bar = off_chan + chan_bytes;
                    const uint32_t nbars = 2 * p.raw_stages + 2 * stages + 2 * b_stages + 2 * kMaxAccGroups + 1;
                    // TMEM slot and stage words, then one 16-byte tile record per raw stage
                    const uint32_t off_rec = round_up(off_bar + nbars * 8 + 4 + 4 * kMaxStages, 16);
                    const uint32_t total = off_rec + 16 * p.raw_stages;
                    if (total > static_cast<uint32_t>(kMaxSmem)) continue;
                    p.cs = cs;
                    p.nslab = p.c_pad / cs;
                    p.stages = stages;
                    p.b_stages = b_stages;
                    p.b_resident = resident;
                    p.b_tile_bytes = b_tile;
                    p.copy_bytes = copy_bytes;
                    p.stage_bytes = stage_bytes;
                    p.off_raw = off_raw;
                    p.off_stages = off_stages;
                    p.off_chan = off_chan;
                    p.off_bar = off_bar;
                    p.off_rec = off_rec;
                    p.smem_bytes = total;
                    break;
                }
                if (p.cs) break;
            }
            if (p.cs) break;
        }
    }
    if (!p.cs) return p;
    {
        // chunks hold whole taps (every k-step of a tap goes to one accumulator)
        const int ksteps = p.cs / (2 * kch), units = p.mmas_per_tile / ksteps;
        const int limit_units = std::max(1, p.limit_mmas / ksteps);
        int nch = (units + limit_units - 1) / limit_units;
        const int per = (units + nch - 1) / nch;
        p.nchunks = (units + per - 1) / per;
        p.chunk_mmas = per * ksteps;
    }
    // Accumulator groups: a tile's chunks go to grp_chunks TMEM buffers that
    // complete together (one hand-off per group).  When two groups of all the
    // tile's chunks do not fit in the 512 columns, a tile takes several groups
    // and carries its running integer sums in NT more columns.
    int sum_cols = 0;
    if (2 * p.nchunks * p.nt <= 512) {
        p.grp_chunks = p.nchunks;
        p.nsg = 1;
    } else {
        p.grp_chunks = std::max(1, (512 - p.nt) / (2 * p.nt));
        p.nsg = (p.nchunks + p.grp_chunks - 1) / p.grp_chunks;
        sum_cols = p.nt;
    }
    p.ngroups = std::min(kMaxAccGroups, (512 - sum_cols) / (p.grp_chunks * p.nt));
    p.tmem_cols = 32;
    while (p.tmem_cols < static_cast<uint32_t>(p.ngroups * p.grp_chunks * p.nt + sum_cols)) p.tmem_cols *= 2;
    p.tiles_per_img = static_cast<int>(p.strip ? strip_tiles : rm_tiles);
    p.total_tiles = static_cast<long long>(p.n_ntiles) * s.n * p.tiles_per_img;
    if (p.total_tiles >= (1ll << 31)) return p;
    p.workspace_bytes = chan_offset(p) + static_cast<size_t>(mp) * (32 + 4 * kThrStride);
    p.ok = true;
    return p;
}

}  // namespace

TcPlan plan_conv_tc(const ConvShape &s)
{
    if (s.bits != 8 && s.c % 32 == 0) {
        // e4m3 staging runs on the converter's fast path only: at most one
        // 16-channel item per thread and slab, strips or kernels at most 5 wide
        const TcPlan p = plan_layout(s, true);
        const int ncol_w = p.strip ? p.sp : s.w;
        if (p.ok && ncol_w * (p.cs / 16) <= 128 && (p.strip || s.kw <= 5)) return p;
    }
    return plan_layout(s, false);
}

cudaError_t launch_conv_tc_prep(const TcPlan &plan, const ConvShape &s, const ConvParams &p, void *workspace,
                                cudaStream_t st)
{
    uint16_t *wpack = static_cast<uint16_t *>(workspace);
    int4 *chan = reinterpret_cast<int4 *>(static_cast<uint8_t *>(workspace) + chan_offset(plan));
    const int mp = plan.n_ntiles * plan.nt;
    int32_t *thr = reinterpret_cast<int32_t *>(chan + 2 * mp);
#define QNN_PREP(B)                                                                                              \
    conv_tc_prep_kernel<B><<<(mp + 7) / 8, 256, 0, st>>>(p.w, p.bias, p.kappa, p.lambda, p.shifts, p.shift, s.m, \
                                                         mp, s.kh, s.kw, s.c, plan.c_pad, plan.k_pad, plan.nt,   \
                                                         plan.nchunks, plan.fp8, wpack, chan, p.thresholds, thr)
    switch (s.bits) {
        case 8: QNN_PREP(8); break;
        case 4: QNN_PREP(4); break;
        default: QNN_PREP(2); break;
    }
#undef QNN_PREP
    return cudaGetLastError();
}

cudaError_t launch_conv_tc_run(const TcPlan &plan, const ConvShape &s, const uint8_t *x, uint8_t *y,
                               const void *workspace, cudaStream_t st, bool after_prep)
{
    if (s.n == 0) return cudaSuccess;
    TcArgs a{};
    a.x = x;
    a.y = y;
    a.wpack = static_cast<const uint8_t *>(workspace);
    a.chan = reinterpret_cast<const int4 *>(static_cast<const uint8_t *>(workspace) + chan_offset(plan));
    a.thr = s.thr ? reinterpret_cast<const int32_t *>(a.chan + 2 * plan.n_ntiles * plan.nt) : nullptr;
    a.off_thr = plan.off_chan + round_up(static_cast<uint32_t>(plan.n_ntiles * plan.nt) * 32 + plan.n_ntiles * plan.nt / 16, 16);
    a.n = s.n; a.h = s.h; a.w = s.w; a.c = s.c; a.m = s.m; a.kh = s.kh; a.kw = s.kw;
    a.ph = s.ph; a.pw = s.pw; a.oh = s.oh; a.ow = s.ow;
    a.c_pad = plan.c_pad; a.cs = plan.cs; a.nslab = plan.nslab;
    a.fp8 = plan.fp8;
    a.kch = plan.fp8 ? 16 : 8;
    {
        const int groups = plan.cs / a.kch;  // K-chunks per slab
        a.log2_groups = groups == 8 ? 3 : groups == 4 ? 2 : 1;
    }
    a.n_ntiles = plan.n_ntiles; a.tiles_per_img = plan.tiles_per_img;
    a.total_tiles = static_cast<int>(plan.total_tiles);
    a.rows_max = plan.rows_max; a.p_alloc = plan.p_alloc;
    a.stages = plan.stages; a.raw_stages = plan.raw_stages; a.b_stages = plan.b_stages;
    a.b_resident = plan.b_resident;
    a.mmas_per_tile = plan.mmas_per_tile; a.chunk_mmas = plan.chunk_mmas; a.nchunks = plan.nchunks;
    a.grp_chunks = plan.grp_chunks; a.ngroups = plan.ngroups; a.nsg = plan.nsg;
    a.row_bytes = plan.row_bytes; a.raw_bytes = plan.raw_bytes;
    a.b_bytes = plan.b_bytes; a.b_tile_bytes = plan.b_tile_bytes;
    a.copy_bytes = plan.copy_bytes; a.stage_bytes = plan.stage_bytes;
    a.chunk_stride = plan.p_alloc * 16;
    a.off_raw = plan.off_raw; a.off_stages = plan.off_stages; a.off_chan = plan.off_chan;
    a.off_bar = plan.off_bar;
    a.off_rec = plan.off_rec;
    a.tmem_cols = plan.tmem_cols;
    a.fd_per_nt = make_fastdiv(static_cast<uint32_t>(s.n * plan.tiles_per_img));
    a.fd_tpi = make_fastdiv(static_cast<uint32_t>(plan.tiles_per_img));
    a.fd_ow = make_fastdiv(static_cast<uint32_t>(s.ow));
    a.strip = plan.strip;
    a.ncb = plan.ncb;
    a.sp = plan.sp;
    a.ncol_w = plan.strip ? plan.sp : s.w;
    a.fd_w = make_fastdiv(static_cast<uint32_t>(a.ncol_w));
    a.fd_ncb = make_fastdiv(static_cast<uint32_t>(std::max(1, plan.ncb)));
    a.a_sbo = plan.strip ? static_cast<uint32_t>(plan.sp) * 16 : 128;
    a.d0_mask = plan.strip ? 0u : 0xFFFFu;
    a.conv_fast = s.c % 8 == 0 && (a.ncol_w << a.log2_groups) <= 128 && (plan.strip || s.kw <= 5);
    a.pool = s.pool;
    a.pool_oh = s.oh / 2;
    a.pool_ow = s.ow / 2;
    // two MMA issuers when every tile of the kernel uses the same resident filter set
    a.mma_warps = (plan.b_resident && plan.nslab == 1 && plan.n_ntiles == 1) ? 2 : 1;
    for (int i = 0; i < s.kh; ++i)
        for (int j = 0; j < s.kw; ++j)
            a.tap_a16[i * s.kw + j] = plan.strip ? static_cast<uint32_t>(i * plan.sp + j)
                                                 : (j * plan.copy_bytes) / 16 + static_cast<uint32_t>(i * s.ow);
    a.status = device_status_ptr();
    if (!a.status) return cudaErrorInvalidSymbol;
    const long long sms = device_sm_count();
    const int grid = static_cast<int>(std::min<long long>(plan.total_tiles, sms));
    switch (s.bits) {
        case 8: return launch_tc_bits<8>(plan.nt, a, grid, plan.smem_bytes, st, after_prep);
        case 4: return launch_tc_bits<4>(plan.nt, a, grid, plan.smem_bytes, st, after_prep);
        default: return launch_tc_bits<2>(plan.nt, a, grid, plan.smem_bytes, st, after_prep);
    }
}

}  // namespace qnn
