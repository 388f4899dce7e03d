// Host-side bounds of the window planner, qnn::plan_conv_win (exported by
// libqnn).  For each layer shape below, every address the window kernel
// derives from a plan (restated here from the kernel's addressing rules) is
// checked against the buffers the plan sizes, for every tile of one image:
//   - shared memory: filters, staged windows, raw windows, records,
//     thresholds, tap sums, barriers, in that order, within 227 KB, with the
//     alignments bulk copies and MMA descriptors need;
//   - every bulk copy of the loader (size, 16-byte alignment of both ends,
//     inside its raw stage and inside the input tensor);
//   - every converter load (inside the bytes the loader copied for that row,
//     and the global element it stands for is the window pixel's) and store
//     (inside its stage);
//   - every A row an MMA reads (inside the staged window, and holding the
//     input pixel that output pixel and tap need), every B row;
//   - tensor memory: one slot of accumulators within 512 columns;
//   - exactness: the planner's worst-case chunk count keeps every chunk within
//     2^22, and its even tap split has no empty chunk;
//   - the reciprocal division the kernel uses for tile and window indices.
// The shapes are the parity tests' and the workloads', then 300 seeded random
// ones across the planner's range.  Prints one line per plan and "fails=N";
// exits non-zero on any failure.
#include <algorithm>
#include <cstdint>
#include <cstdio>
#include <vector>

#include "../paper_1908_11263_gb300/csrc/internal.h"

using namespace qnn;

static int fails = 0;
#define CHECK(c, ...)                                \
    do {                                             \
        if (!(c)) {                                  \
            ++fails;                                 \
            std::printf("FAIL %s: ", #c);            \
            std::printf(__VA_ARGS__);                \
            std::printf("\n");                       \
        }                                            \
    } while (0)

// Constants of the kernel (conv_win.cuh).
static constexpr int kRows = 16, kCols = 8, kConvThreads = 128, kMaxKP = 5, kMaxStages = 4, kMaxSlots = 4;
static constexpr long long kSmemLimit = 232448;
static constexpr long long kBarBytes = (4 * kMaxStages + 2 * kMaxSlots + 3) * 8 + 32;

// The kernel's reciprocal division: floor(n * m / 2^64), m = ceil(2^64 / d).
static int fdiv(long long n, unsigned d)
{
    if (d <= 1) return static_cast<int>(n);
    const unsigned long long m = (~0ull / d) + 1ull;
    return static_cast<int>((static_cast<unsigned __int128>(static_cast<unsigned long long>(n)) * m) >> 64);
}

static void check(int n, int h, int w, int c, int m, int kh, int kw, int ph, int pw, int bits, int pool)
{
    ConvShape s{};
    s.n = n; s.h = h; s.w = w; s.c = c; s.m = m; s.kh = kh; s.kw = kw; s.sh = 1; s.sw = 1;
    s.ph = ph; s.pw = pw; s.bits = bits; s.pool = pool; s.thr = 0;
    s.oh = h + 2 * ph - kh + 1;
    s.ow = w + 2 * pw - kw + 1;
    if (pool && (s.oh < 2 || s.ow < 2)) return;  // qconv_hwc_pool2 rejects these before planning
    const WinPlan p = plan_conv_win(s);
    std::printf("%dx%dx%dx%d->%d k%dx%d p%d,%d q%d pool%d: ok=%d", n, h, w, c, m, kh, kw, ph, pw, bits, pool, p.ok);
    if (!p.ok) {
        std::printf("\n");
        return;
    }
    std::printf(" S=%d %s nt=%d sp=%d wh=%d stages=%d/%d nch=%d..%d smem=%u wcopy=%u %s%s\n", p.s,
                p.fp8 ? "e4m3" : "fp16", p.nt, p.sp, p.wh, p.a_stages, p.raw_stages, p.nch_min, p.nch_max, p.smem_bytes,
                p.wraw_bytes, p.full_rows ? "full-rows" : "row-segments", p.fold ? " folded" : "");
    // folded plans: a tap is a kernel row, a position holds kw pixels' c channels
    CHECK(p.fold == (bits == 8 && c % 8 != 0 && kw > 1 && c * kw <= 16 && m <= 64), "fold rule");
    CHECK(p.fold ? (p.taps == kh && p.kwf == 1 && p.groups == 2 && p.c_pad == 16 && p.full_rows &&
                    p.sp == kCols * p.s)
                 : (p.taps == kh * kw && p.kwf == kw && p.sp == kCols * p.s + kw - 1),
          "fold layout");
    const long long cb = static_cast<long long>(c) * bits / 8;
    const int kch = p.fp8 ? 16 : 8, gbytes = kch * bits / 8;  // packed bytes of one K-chunk
    CHECK(gbytes == (bits == 8 ? 8 : 16 * bits / 8), "gbytes %d", gbytes);
    const int npos = p.wh * p.sp;
    // shared memory layout
    const long long rec_bytes = 2LL * p.nt * 16 + p.nt / 16;
    CHECK(p.off_b == 0 && p.off_b + p.b_bytes <= p.off_a, "filters");
    CHECK(p.off_a % 128 == 0 && p.off_a + static_cast<long long>(p.a_stages) * p.stage_bytes <= p.off_raw, "stages");
    CHECK(p.off_raw % 128 == 0 && p.off_raw + static_cast<long long>(p.raw_stages) * p.raw_bytes <= p.off_rec, "raw");
    CHECK(p.off_rec % 16 == 0 && p.off_rec + rec_bytes <= p.off_thr, "records");
    CHECK(p.off_tap + (p.taps + 3LL) * p.nt * 4 <= p.off_mtab && p.off_tap % 4 == 0, "tap sums");
    CHECK(p.off_mtab % 8 == 0 && p.off_mtab + 8LL * p.s * p.taps * p.ksteps <= p.off_pre, "MMA table");
    CHECK(p.off_pre % 128 == 0 && p.off_pre + 4096LL + 32LL * p.nt <= p.off_wraw, "pre-load operands");
    CHECK(p.off_wraw % 16 == 0 && p.off_wraw + p.wraw_bytes <= p.off_bar, "filter copy");
    if (p.wraw_bytes) CHECK(p.wraw_bytes == static_cast<long long>(m) * kh * kw * cb && p.wraw_bytes % 16 == 0,
                            "filter copy size");
    CHECK(p.off_bar % 16 == 0 && p.off_bar + kBarBytes <= p.smem_bytes && p.smem_bytes <= kSmemLimit, "barriers");
    // the MMA issue table the filter preparation writes, for every chunk count the kernel
    // can take: each entry written once, inside the table, and every (tap, k-step, strip)
    // issued once into the accumulator of its chunk
    for (int nch = p.nch_min; nch <= std::max(p.nch_min, p.nch_max); ++nch) {
        const int ct = (p.taps + nch - 1) / nch, last_len = p.taps - (nch - 1) * ct;
        if (last_len <= 0) continue;  // the kernel never takes a split with an empty chunk
        const int nmma = p.s * p.taps * p.ksteps;
        // K-split (the kernel's rule): k-step kk of a tap goes to accumulator kk % kx of its chunk
        const int kx = (p.s * nch == 1 && p.ksteps % 2 == 0 && 2 * p.nt <= 256) ? 2 : 1;
        CHECK(p.s * nch * kx * p.nt <= 512, "slot with the K-split");
        std::vector<int> seen(nmma, 0), unit(p.taps * p.ksteps * p.s, 0);
        CHECK(ct * p.ksteps <= 256, "one step pair per preparation thread");
        for (int et = 0; et < ct * p.ksteps; ++et) {
            const int jt = et / p.ksteps, kk = et - jt * p.ksteps;
            const int nj = jt < last_len ? nch : nch - 1;
            const int before = jt * nch - std::max(0, jt - last_len);
            int u = p.s * (p.ksteps * before + kk * nj);
            for (int cc = 0; cc < nj; ++cc) {
                const int tap = cc * ct + jt;
                CHECK(tap < p.taps, "table tap");
                for (int sj = 0; sj < p.s; ++sj, ++u) {
                    CHECK(u >= 0 && u < nmma, "table index %d", u);
                    if (u >= 0 && u < nmma) ++seen[u];
                    ++unit[(tap * p.ksteps + kk) * p.s + sj];
                    CHECK(((sj * nch + cc) * kx + kk % kx) * p.nt + p.nt <= p.s * nch * kx * p.nt, "accumulator column");
                    CHECK(8LL * nmma <= 8LL * p.s * p.taps * p.ksteps, "table size");
                }
            }
        }
        for (int u = 0; u < nmma; ++u) CHECK(seen[u] == 1, "table entry %d written %d times", u, seen[u]);
        for (size_t q = 0; q < unit.size(); ++q) CHECK(unit[q] == 1, "MMA unit %zu issued %d times", q, unit[q]);
    }
    // MMA table entries: A offset in 16 bits, accumulator column below 512 in the upper 16
    {
        const long long a_max = (kh - 1LL) * p.sp + (kw - 1) + (p.ksteps - 1LL) * 2 * (p.chunk_stride / 16) + kCols;
        CHECK(a_max < 65536, "A offset field");
        const int cf = std::max(p.nch_min, p.nch_max);
        CHECK((p.s * cf - 1LL) * p.nt < 512, "accumulator field");
    }
    CHECK(p.a_stages >= 2 && p.a_stages <= kMaxStages && p.raw_stages >= 2 && p.raw_stages <= kMaxStages, "rings");
    CHECK(p.raw_bytes % 16 == 0 && p.stage_bytes % 16 == 0 && p.chunk_stride % 16 == 0, "16-byte units");
    CHECK(p.chunk_stride >= static_cast<unsigned>(npos) * 16 && p.stage_bytes == p.chunk_stride * p.groups, "planes");
    // MMA descriptors: 14-bit fields of 16-byte units
    CHECK(p.smem_bytes < (1u << 18) && p.chunk_stride < (1u << 18) && p.sp * 16 < (1 << 18), "descriptor fields");
    CHECK(p.groups % 2 == 0 && p.ksteps * 2 == p.groups && p.groups <= 8, "k-steps");
    // converter positions
    CHECK(npos <= kMaxKP * kConvThreads, "npos %d", npos);
    // tensor memory and exactness
    CHECK(p.s * p.nch_max * p.nt <= 512, "tmem");
    const long long max_prod = p.fp8 ? (bits == 4 ? 15 * 8 : 3 * 2) : 128 * 128;
    {
        const int ct = (p.taps + p.nch_max - 1) / p.nch_max;
        CHECK(static_cast<long long>(ct) * p.c_pad * max_prod <= (1LL << 22), "worst-case chunk");
        CHECK((p.nch_max - 1) * ct < p.taps, "empty chunk");
        // the chunk count the kernel forces whatever the filters: valid by the same bound
        const int cf = std::max(p.nch_min, p.nch_max), cft = (p.taps + cf - 1) / cf;
        CHECK(p.nch_min >= 1 && (cf - 1) * cft < p.taps, "forced chunk count %d", cf);
        CHECK(static_cast<long long>(cft) * p.c_pad * max_prod <= (1LL << 22), "forced chunk bound");
        CHECK(p.s * cf * p.nt <= 512, "tmem at the forced chunk count");
    }
    CHECK(256 % p.nt == 0 && p.nt >= m, "prep channel per thread");
    // the filter-prep loads: the last K-chunk of the last channel inside the packed filters
    // (folded: the bytes of a kernel row, kw * c of them, read one by one)
    if (p.fold)
        CHECK((static_cast<long long>(m - 1) * p.taps + p.taps - 1) * kw * c + kw * c <=
                  static_cast<long long>(m) * kh * kw * c && kw * c <= 16,
              "prep loads (folded)");
    else
        CHECK((static_cast<long long>(m - 1) * p.taps + p.taps - 1) * cb + (c * bits / 8 / gbytes - 1) * gbytes +
                      gbytes <=
                  static_cast<long long>(m) * p.taps * cb,
              "prep loads");
    CHECK(p.taps * p.groups * p.nt * 16LL == p.b_bytes, "B size");
    // division used for window positions
    for (int pos = 0; pos < kMaxKP * kConvThreads; ++pos) CHECK(fdiv(pos, p.sp) == pos / p.sp, "fdiv sp %d", pos);
    // every tile of the first and the last image
    const long long x_bytes = static_cast<long long>(n) * h * w * cb;
    for (int img : {0, n - 1}) {
        for (int ti = 0; ti < p.tiles_per_img; ++ti) {
            const long long t = static_cast<long long>(img) * p.tiles_per_img + ti;
            const int gi = fdiv(t, p.tiles_per_img);
            CHECK(gi == img, "fdiv tile");
            const int ty = fdiv(ti, p.tiles_x), tx = ti - ty * p.tiles_x;
            const int oy0 = ty * kRows, ox0 = tx * kCols * p.s, iy0 = oy0 - ph, ix0 = ox0 - pw;
            const int r0 = std::min(p.wh, std::max(0, -iy0)), r1 = std::max(r0, std::min(p.wh, h - iy0));
            const int c0 = std::min(p.sp, std::max(0, -ix0)), c1 = std::max(c0, std::min(p.sp, w - ix0));
            // loader
            const long long seg = p.full_rows ? static_cast<long long>(w) * cb : (c1 - c0) * cb;
            CHECK(static_cast<long long>(r1 - r0) * p.raw_row_bytes <= p.raw_bytes, "raw stage rows");
            CHECK(seg <= p.raw_row_bytes && seg % 16 == 0 && p.raw_row_bytes % 16 == 0, "copy size");
            for (int r = r0; r < r1; ++r) {
                const long long src =
                    ((static_cast<long long>(img) * h + iy0 + r) * w + (p.full_rows ? 0 : ix0 + c0)) * cb;
                CHECK(src >= 0 && src + seg <= x_bytes && src % 16 == 0, "copy source row %d", r);
                CHECK(iy0 + r >= 0 && iy0 + r < h, "copied row inside the image");
            }
            if (p.full_rows && !p.fold) CHECK(ix0 + c0 == 0 && ix0 + c1 == w, "whole rows");
            if (p.fold) {
                // folded converter: whole image rows; a position inside the image in both
                // directions reads five aligned words from its row's first byte, rounded
                // down to 4; the words stay inside shared memory, the span inside the row
                for (int pos = 0; pos < npos; ++pos) {
                    const int r = fdiv(pos, p.sp), px = pos - r * p.sp, colx = ix0 + px;
                    CHECK(2LL * p.chunk_stride <= p.stage_bytes && pos * 16LL + 16 <= p.chunk_stride, "folded store");
                    if (r < r0 || r >= r1) {
                        CHECK(iy0 + r < 0 || iy0 + r >= h, "folded row outside the image");
                        continue;
                    }
                    CHECK(iy0 + r >= 0 && iy0 + r < h, "folded row inside the image");
                    // the span's pixels inside the image, [jlo, jhi): their bytes from the first one on
                    const int jlo = std::max(0, -colx), jhi = std::min(kw, w - colx);
                    if (jhi <= jlo) continue;
                    const long long off = static_cast<long long>(colx + jlo) * c;
                    const long long word0 = static_cast<long long>(r - r0) * p.raw_row_bytes + (off & ~3LL);
                    CHECK(off >= 0 && off + (jhi - jlo) * c <= static_cast<long long>(w) * c, "folded span inside the row");
                    CHECK(jlo * c * 8 < 128 && jhi * c <= 16, "folded shift and mask");
                    CHECK(p.raw_row_bytes % 4 == 0 &&
                              p.off_raw + static_cast<long long>(p.raw_stages - 1) * p.raw_bytes + word0 + 20 <=
                                  p.smem_bytes,
                          "folded word loads");
                }
                for (int sj = 0; sj < p.s; ++sj)
                    for (int i = 0; i < kh; ++i)
                        for (int g = 0; g < kRows; ++g)
                            for (int col = 0; col < kCols; ++col) {
                                const int pos = i * p.sp + sj * kCols + g * p.sp + col;
                                CHECK(pos >= 0 && pos < npos, "folded A row");
                                const int r = pos / p.sp, px = pos % p.sp;
                                const int oy = oy0 + g, ox = ox0 + sj * kCols + col;
                                if (oy < s.oh && ox < s.ow)
                                    CHECK(iy0 + r == oy - ph + i && ix0 + px == ox - pw, "folded A row pixels");
                            }
                for (int tap = 0; tap < p.taps; ++tap)
                    CHECK((static_cast<long long>(tap) * p.groups + 2) * p.nt * 16 <= p.b_bytes, "folded B rows");
                continue;
            }
            // converter
            const int base_col = p.full_rows ? ix0 : -c0;
            for (int tid = 0; tid < kConvThreads; ++tid)
                for (int k = 0; k < kMaxKP; ++k) {
                    const int pos = tid + 128 * k;
                    if (pos >= npos) continue;
                    const int r = fdiv(pos, p.sp), px = pos - r * p.sp;
                    const bool ok = r >= r0 && r < r1 && px >= c0 && px < c1;
                    const bool inside = iy0 + r >= 0 && iy0 + r < h && ix0 + px >= 0 && ix0 + px < w;
                    CHECK(ok == inside, "staged pixel inside the image");
                    for (int gq = 0; gq < p.groups; ++gq)
                        CHECK(static_cast<long long>(gq) * p.chunk_stride + pos * 16LL + 16 <= p.stage_bytes, "store");
                    // one pixel's packed channels, in 16-byte loads when the pixel is whole
                    // 16-byte units, else 8-byte ones (a padding position reads the stage's
                    // first bytes instead)
                    const int unit = cb % 16 == 0 ? 16 : 8;
                    CHECK(cb % 8 == 0 && cb <= 64, "pixel bytes");
                    CHECK(cb <= static_cast<long long>(p.raw_bytes), "padding load");
                    if (!ok) continue;
                    const long long src = static_cast<long long>(r - r0) * p.raw_row_bytes + (px + base_col) * cb;
                    CHECK(src >= 0 && src + cb <= static_cast<long long>(r1 - r0) * p.raw_row_bytes, "raw load");
                    // byte q of copied row r stands for global byte row_start + q
                    const long long row_start =
                        ((static_cast<long long>(img) * h + iy0 + r) * w + (p.full_rows ? 0 : ix0 + c0)) * cb;
                    const long long q = src - static_cast<long long>(r - r0) * p.raw_row_bytes;
                    CHECK(q + cb <= seg, "inside the copied span");
                    const long long want = ((static_cast<long long>(img) * h + iy0 + r) * w + ix0 + px) * cb;
                    CHECK(row_start + q == want, "the pixel's own channels");
                    CHECK(src % unit == 0 && p.raw_row_bytes % 16 == 0, "load alignment");
                }
            // MMA A rows and B rows
            for (int sj = 0; sj < p.s; ++sj)
                for (int i = 0; i < kh; ++i)
                    for (int j = 0; j < kw; ++j)
                        for (int g = 0; g < kRows; ++g)
                            for (int col = 0; col < kCols; ++col) {
                                const int pos = i * p.sp + j + sj * kCols + g * p.sp + col;
                                CHECK(pos >= 0 && pos < npos, "A row");
                                const int r = pos / p.sp, px = pos % p.sp;
                                const int oy = oy0 + g, ox = ox0 + sj * kCols + col;
                                if (oy < s.oh && ox < s.ow)
                                    CHECK(iy0 + r == oy - ph + i && ix0 + px == ox - pw + j, "A row pixel");
                            }
            for (int tap = 0; tap < p.taps; ++tap)
                for (int kk = 0; kk < p.ksteps; ++kk)
                    CHECK((static_cast<long long>(tap) * p.groups + 2 * kk + 2) * p.nt * 16 <= p.b_bytes, "B rows");
        }
    }
}

int main()
{
    // n, h, w, c, m, kh, kw, ph, pw, bits: the parity tests' shapes and the workloads'
    static const int shapes[][10] = {
        {2, 16, 16, 32, 64, 3, 3, 1, 1, 8},     {1, 16, 16, 32, 64, 3, 3, 1, 1, 4},   {1, 16, 16, 32, 64, 3, 3, 1, 1, 2},
        {3, 10, 10, 16, 16, 3, 3, 1, 1, 8},     {2, 14, 14, 64, 48, 3, 3, 1, 1, 8},   {1, 15, 20, 24, 40, 3, 3, 1, 1, 8},
        {1, 12, 12, 3, 32, 5, 5, 2, 2, 8},      {2, 8, 8, 32, 64, 5, 5, 2, 2, 8},     {1, 7, 7, 128, 136, 3, 3, 1, 1, 8},
        {1, 6, 6, 256, 256, 3, 3, 1, 1, 8},     {1, 5, 9, 32, 16, 3, 2, 0, 1, 8},     {1, 11, 13, 16, 32, 2, 4, 1, 2, 8},
        {1, 1, 40, 16, 16, 1, 3, 0, 1, 8},      {2, 13, 13, 32, 24, 3, 3, 0, 0, 4},   {1, 10, 12, 48, 32, 5, 5, 2, 2, 4},
        {2, 9, 9, 64, 64, 3, 3, 1, 1, 2},       {1, 9, 7, 8, 12, 3, 3, 1, 1, 2},      {1, 16, 16, 12, 16, 3, 3, 1, 1, 4},
        {512, 16, 16, 32, 64, 3, 3, 1, 1, 8},   {512, 16, 16, 32, 64, 3, 3, 1, 1, 4}, {512, 16, 16, 32, 64, 3, 3, 1, 1, 2},
        {1024, 32, 32, 3, 32, 5, 5, 2, 2, 8},   {1024, 16, 16, 32, 32, 5, 5, 2, 2, 8}, {1024, 8, 8, 32, 64, 5, 5, 2, 2, 8},
        {64, 56, 56, 64, 64, 3, 3, 1, 1, 8},    {64, 28, 28, 128, 128, 3, 3, 1, 1, 8}, {64, 14, 14, 256, 256, 3, 3, 1, 1, 8},
        {64, 14, 14, 256, 512, 1, 1, 0, 0, 8},  {1, 4, 32, 256, 16, 1, 1, 0, 0, 8},   {1, 6, 6, 256, 32, 3, 3, 1, 1, 4},
        {1, 8, 8, 32, 32, 3, 3, 1, 1, 8},       {2, 30, 16, 32, 64, 3, 3, 1, 1, 8},   {1, 16, 24, 32, 48, 5, 5, 2, 2, 8},
        {1, 47, 40, 32, 32, 3, 3, 1, 1, 4},     {1, 47, 40, 64, 32, 3, 3, 1, 1, 2},   {3, 9, 11, 16, 16, 1, 1, 0, 0, 8},
        {2, 32, 32, 3, 32, 5, 5, 2, 2, 8},      {1, 12, 12, 32, 136, 3, 3, 1, 1, 8},  {1, 14, 22, 32, 32, 3, 3, 1, 1, 2},
        {1, 16, 16, 32, 64, 3, 3, 1, 1, 8},     {2, 20, 36, 32, 64, 3, 3, 1, 1, 8},   {1, 17, 40, 64, 128, 7, 7, 3, 3, 8},
        {1, 9, 24, 128, 96, 3, 3, 1, 1, 4},     {1, 9, 24, 128, 96, 3, 3, 1, 1, 2},   {2, 3, 3, 32, 32, 3, 3, 1, 1, 8},
        {1, 16, 16, 64, 64, 3, 3, 1, 1, 8},     {1, 24, 40, 32, 32, 5, 5, 2, 2, 8},   {3, 18, 18, 16, 16, 3, 3, 0, 0, 8},
        {2, 21, 32, 3, 16, 3, 3, 1, 1, 8},      {1, 16, 48, 5, 24, 3, 3, 1, 1, 8},    {2, 19, 16, 1, 8, 7, 7, 3, 3, 8},
        {1, 20, 32, 2, 40, 5, 5, 0, 0, 8},      {3, 9, 16, 4, 32, 4, 4, 2, 1, 8},
    };
    for (const auto &v : shapes) check(v[0], v[1], v[2], v[3], v[4], v[5], v[6], v[7], v[8], v[9], 0);
    for (const auto &v : shapes) check(v[0], v[1], v[2], v[3], v[4], v[5], v[6], v[7], v[8], v[9], 1);
    // seeded random shapes across the planner's range (whatever it accepts is checked)
    unsigned long long rng = 0x5EEDB0D5ull;
    auto next = [&](int lo, int hi) {  // uniform in [lo, hi]
        rng = rng * 6364136223846793005ull + 1442695040888963407ull;
        return lo + static_cast<int>((rng >> 33) % static_cast<unsigned long long>(hi - lo + 1));
    };
    for (int i = 0; i < 300; ++i) {
        static const int kBits[4] = {8, 8, 4, 2};
        const int bits = kBits[next(0, 3)];
        const int per = 8 / bits;
        const int c = bits == 8 ? (next(0, 3) == 0 ? next(1, 7) : 8 * next(1, 8)) : 32 * next(1, bits == 4 ? 4 : 8);
        const int m = per * next(1, 128 / per);
        const int kh = next(1, 7), kw = next(1, 7);
        const int ph = next(0, kh / 2), pw = next(0, kw / 2);
        const int h = next(std::max(1, kh - 2 * ph), 40), w = next(std::max(1, kw - 2 * pw), 48);
        check(next(1, 3), h, w, c, m, kh, kw, ph, pw, bits, next(0, 1));
    }
    std::printf("fails=%d\n", fails);
    return fails ? 1 : 0;
}
