// Host-side bounds of the tensor-core planner, qnn::plan_conv_tc (exported by
// libqnn).  For each layer shape below, the addresses the kernel derives from
// a plan (restated here from the kernel's addressing rules) are checked
// against the buffers the plan sizes:
//   - shared memory: the filter region, the raw-row ring, the staged A
//     stages, the per-channel records, the barriers and the tile records, in
//     that order, within the 227 KB a CTA may use;
//   - every converter store and every raw-row load of every tile, for each
//     of the 128 converter threads' fixed column items (row tiles and strips);
//   - every A row an MMA reads, and that the rows feeding stored outputs hold
//     the input pixels the convolution needs;
//   - tensor memory: accumulator groups within 512 columns;
//   - exactness: no accumulator chunk can reach 2^22 in magnitude;
//   - the reciprocal division the kernel uses for tile indices.
// Prints one line per plan and "fails=N"; exits non-zero on any failure.
#include <algorithm>
#include <cstdint>
#include <cstdio>

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

static constexpr int kTileM = 128, kThreads = 128;  // MMA rows per tile; converter threads
static constexpr int kMaxAccGroups = 4, kMaxStages = 4;
static constexpr long long kMaxSmem = 232448;

// The converter's fixed column items: thread t takes items ci0, ci0 + cstep, ...
// of `ncol` and rows rp, rp + nphase, ... (the kernel's conv_map).
struct Items {
    int nphase, rp, ci0, cstep;
};
static Items items(int ncol, int t)
{
    Items m;
    if (ncol <= kThreads) {
        m.nphase = kThreads / ncol;
        m.rp = t / ncol;
        m.ci0 = m.rp < m.nphase ? t - m.rp * ncol : ncol;
        m.cstep = ncol;
        if (m.rp >= m.nphase) m.rp = 0;
    } else {
        m.nphase = 1;
        m.rp = 0;
        m.ci0 = t;
        m.cstep = kThreads;
    }
    return m;
}

// Raw-row window of a tile starting at output row oy0: staged rows [r_lo, r_hi) lie in the image.
static void window(int rows, int oy0, int ph, int h, int *r_lo, int *r_hi)
{
    const int iy0 = oy0 - ph;
    *r_lo = std::min(rows, std::max(0, -iy0));
    *r_hi = std::max(*r_lo, std::min(rows, h - iy0));
}

static int load_bytes(const TcPlan &p, int bits)
{
    if (p.fp8) return bits == 4 ? 8 : 4;  // 16 channels as e4m3 sources
    return bits == 8 ? 8 : bits == 4 ? 4 : 2;  // 8 channels
}

static void check_strip(const ConvShape &s, const TcPlan &p, int kch)
{
    const int groups = p.cs / kch, sp = p.sp;
    CHECK(sp == 8 + s.kw - 1 && p.ncb == (s.ow + 7) / 8 && p.tiles_per_img == p.ncb * ((s.oh + 15) / 16),
          "strip dims");
    CHECK((long long)groups * p.p_alloc * 16 <= p.stage_bytes && p.stage_bytes == p.copy_bytes, "strip stage");
    // MMA: tap (i, j), row group g, row q of the group reads window position (g + i) * sp + j + q
    CHECK((15 + s.kh - 1) * sp + (s.kw - 1) + 7 < p.p_alloc, "strip A reads");
    const int ncol = sp * groups;
    for (int ti = 0; ti < p.tiles_per_img; ++ti) {
        const int rb = ti / p.ncb, oy0 = rb * 16, ox0 = (ti - rb * p.ncb) * 8;
        const int rows = std::min(p.rows_max, s.oh - oy0 + s.kh - 1);
        int r_lo, r_hi;
        window(rows, oy0, s.ph, s.h, &r_lo, &r_hi);
        CHECK(rows > 0 && (long long)(r_hi - r_lo) * p.row_bytes <= p.raw_bytes, "strip raw bytes ti=%d", ti);
        if (r_hi > r_lo) CHECK(oy0 - s.ph + r_lo >= 0 && oy0 - s.ph + r_hi <= s.h, "strip raw rows ti=%d", ti);
        // stored outputs read staged rows only, and the window holds the input pixels they need
        for (int g = 0; g < 16 && oy0 + g < s.oh; ++g)
            for (int q = 0; q < 8 && ox0 + q < s.ow; ++q)
                for (int i = 0; i < s.kh; ++i)
                    for (int j = 0; j < s.kw; ++j) {
                        const int r = g + i, px = q + j;
                        CHECK(r < rows && px < sp, "strip valid read ti=%d", ti);
                        CHECK(oy0 + g - s.ph + i == oy0 - s.ph + r && ox0 + q - s.pw + j == ox0 - s.pw + px,
                              "strip window map");
                    }
        for (int t = 0; t < kThreads; ++t) {
            const Items m = items(ncol, t);
            for (int ci = m.ci0; ci < ncol; ci += m.cstep) {
                const int gq = ci / sp, px = ci - gq * sp;
                CHECK(gq < groups, "strip item");
                for (int slab = 0; slab < p.nslab; ++slab) {
                    const int c0 = slab * p.cs + gq * kch;
                    if (c0 >= s.c) continue;
                    const int ix = ox0 - s.pw + px;
                    const bool col_ok = ix >= 0 && ix < s.w;
                    for (int r = m.rp; r < rows; r += m.nphase) {
                        const long long off = (long long)gq * p.p_alloc * 16 + ((long long)r * sp + px) * 16;
                        CHECK(off >= 0 && off + 16 <= p.stage_bytes, "strip store");
                        if (r >= r_lo && r < r_hi && col_ok && s.c % 8 == 0) {
                            const int lb = load_bytes(p, s.bits);
                            const long long ro = (long long)(r - r_lo) * p.row_bytes +
                                                 (long long)ix * s.c * s.bits / 8 + (long long)c0 * s.bits / 8;
                            CHECK(ro >= 0 && ro + lb <= (long long)(r_hi - r_lo) * p.row_bytes && ro % lb == 0,
                                  "strip load");
                        }
                    }
                }
            }
        }
    }
}

static void check_rows(const ConvShape &s, const TcPlan &p, int kch)
{
    const int groups = p.cs / kch;
    for (int ti = 0; ti < p.tiles_per_img; ++ti) {
        const int p0 = ti * kTileM, oy_a = p0 / s.ow, d0 = p0 - oy_a * s.ow;
        const int out_rows = std::min((d0 + kTileM + s.ow - 1) / s.ow, s.oh - oy_a);
        const int rows = std::min(p.rows_max, out_rows + s.kh - 1);
        int r_lo, r_hi;
        window(rows, oy_a, s.ph, s.h, &r_lo, &r_hi);
        CHECK((long long)(r_hi - r_lo) * p.row_bytes <= p.raw_bytes, "raw bytes ti=%d", ti);
        if (r_hi > r_lo) CHECK(oy_a - s.ph + r_lo >= 0 && oy_a - s.ph + r_hi <= s.h, "raw rows in image ti=%d", ti);
        CHECK(rows * s.ow <= p.p_alloc, "store positions ti=%d rows=%d", ti, rows);
        const int last_valid = std::min(kTileM, s.oh * s.ow - p0) - 1;
        CHECK((d0 + last_valid) / s.ow + s.kh - 1 < rows, "stored pixel reads an unstaged row ti=%d", ti);
        // copy j of tap (i, j), read i * ow positions later: the last of the 128 rows
        CHECK(d0 + (s.kh - 1) * s.ow + kTileM - 1 < p.p_alloc, "A reads ti=%d", ti);
    }
    const int ncol = s.w * groups;
    for (int t = 0; t < kThreads; ++t) {
        const Items m = items(ncol, t);
        for (int ci = m.ci0; ci < ncol; ci += m.cstep) {
            const int gq = ci / s.w, x = ci - gq * s.w;
            CHECK(gq < groups && x < s.w, "column item");
            for (int slab = 0; slab < p.nslab; ++slab) {
                const int c0 = slab * p.cs + gq * kch;
                for (int ti = 0; ti < p.tiles_per_img; ++ti) {
                    const int p0 = ti * kTileM, oy_a = p0 / s.ow, d0 = p0 - oy_a * s.ow;
                    const int out_rows = std::min((d0 + kTileM + s.ow - 1) / s.ow, s.oh - oy_a);
                    const int rows = std::min(p.rows_max, out_rows + s.kh - 1);
                    int r_lo, r_hi;
                    window(rows, oy_a, s.ph, s.h, &r_lo, &r_hi);
                    // copies j in [jlo, jhi] hold pixel x (their column x + pw - j lies in [0, ow))
                    const int jlo = std::max(0, x + s.pw - s.ow + 1), jhi = std::min(s.kw - 1, x + s.pw);
                    const unsigned jmask = jhi >= jlo ? ((2u << jhi) - (1u << jlo)) : 0u;
                    for (int r = m.rp; r < rows; r += m.nphase) {
                        for (int j = 0; j < s.kw; ++j) {
                            const int ox = x + s.pw - j;
                            CHECK(((jmask >> j) & 1u) == (ox >= 0 && ox < s.ow ? 1u : 0u), "copy mask");
                            if (ox < 0 || ox >= s.ow) continue;
                            const long long off = (long long)j * p.copy_bytes + (long long)gq * p.p_alloc * 16 +
                                                  ((long long)r * s.ow + ox) * 16;
                            CHECK(off >= 0 && off + 16 <= p.stage_bytes && r * s.ow + ox < p.p_alloc, "store");
                        }
                        if (r >= r_lo && r < r_hi && c0 < s.c && s.c % 8 == 0) {
                            const int lb = load_bytes(p, s.bits);
                            const long long ro = (long long)(r - r_lo) * p.row_bytes +
                                                 (long long)x * s.c * s.bits / 8 + (long long)c0 * s.bits / 8;
                            CHECK(ro >= 0 && ro + lb <= (long long)(r_hi - r_lo) * p.row_bytes && ro % lb == 0,
                                  "load");
                        }
                    }
                }
            }
        }
    }
    CHECK((long long)(s.kw - 1) * p.copy_bytes + (long long)groups * p.p_alloc * 16 <= p.stage_bytes,
          "stage extent");
}

static void check(int n, int h, int w, int c, int m, int kh, int kw, int ph, int pw, int bits, int pool)
{
    ConvShape s{n, h, w, c, m, kh, kw, 1, 1, ph, pw, bits, h + 2 * ph - kh + 1, w + 2 * pw - kw + 1};
    s.pool = pool;
    const TcPlan p = plan_conv_tc(s);
    std::printf("%dx%dx%dx%d->%d k%dx%d p%d,%d q%d pool%d: ok=%d %s %s nt=%d cs=%d slabs=%d stages=%d smem=%u "
                "tmem=%u chunks=%dx%d\n",
                n, h, w, c, m, kh, kw, ph, pw, bits, pool, p.ok, p.strip ? "strips" : "rows", p.fp8 ? "e4m3" : "fp16",
                p.nt, p.cs, p.nslab, p.stages, p.smem_bytes, p.tmem_cols, p.nchunks, p.chunk_mmas);
    if (!p.ok) return;
    const int kch = p.fp8 ? 16 : 8;  // channels per 16-byte K-chunk
    if (pool) CHECK(p.strip, "the fused pool needs strips");
    CHECK(!p.fp8 || (bits != 8 && c % 32 == 0 && p.c_pad % 32 == 0 && p.cs >= 32), "e4m3 shape");
    // shared-memory layout
    CHECK(p.smem_bytes <= kMaxSmem, "smem");
    if (p.b_resident) {
        const long long chunks = ((long long)(kh * kw - 1) * p.c_pad + (long long)(p.nslab - 1) * p.cs) / kch + p.cs / kch;
        CHECK(chunks * p.nt * 16 <= p.b_bytes && p.b_bytes <= p.off_raw, "resident filters");
    } else {
        CHECK((long long)p.b_stages * p.b_tile_bytes <= p.off_raw &&
                  p.b_tile_bytes == (uint32_t)(p.nt * p.cs * (p.fp8 ? 1 : 2)),
              "streamed filter ring");
    }
    CHECK(p.off_raw + p.raw_stages * p.raw_bytes <= p.off_stages, "raw region");
    CHECK(p.off_stages + p.stages * p.stage_bytes <= p.off_chan, "stage region");
    CHECK(p.off_chan + (uint32_t)(p.n_ntiles * p.nt * 32 + p.n_ntiles * p.nt / 16) <= p.off_bar, "record region");
    const long long bars = 2 * p.raw_stages + 2 * p.stages + 2 * p.b_stages + 2 * kMaxAccGroups + 1;
    CHECK(p.stages <= kMaxStages && p.off_rec % 16 == 0 && p.off_rec >= p.off_bar + bars * 8 + 4 + 4 * kMaxStages &&
              p.off_rec + 16 * p.raw_stages <= p.smem_bytes,
          "barriers and tile records");
    CHECK(p.row_bytes % 16 == 0 && p.raw_bytes % 128 == 0 && p.off_raw % 128 == 0 && p.off_stages % 16 == 0,
          "bulk-copy alignment");
    // exact accumulator chunks and tensor memory
    const long long max_prod = p.fp8 ? (bits == 4 ? 15 * 8 : 3 * 2) : (bits == 8 ? 16384 : bits == 4 ? 1039 * 8 : 1027 * 2);
    CHECK(p.chunk_mmas * p.nchunks >= p.mmas_per_tile, "chunks cover the tile");
    CHECK((long long)p.chunk_mmas * (p.fp8 ? 32 : 16) * max_prod <= (1ll << 22), "exact chunk");
    CHECK(p.ngroups * p.grp_chunks * p.nt + (p.nsg > 1 ? p.nt : 0) <= (int)p.tmem_cols && p.tmem_cols <= 512 &&
              p.ngroups >= 2 && p.ngroups <= kMaxAccGroups && p.nsg * p.grp_chunks >= p.nchunks &&
              (p.nsg - 1) * p.grp_chunks < p.nchunks,
          "tensor memory");
    if (p.strip) check_strip(s, p, kch);
    else check_rows(s, p, kch);
}

// The kernel divides by constants as q = floor(n * ceil(2^64 / d) / 2^64);
// this is exact for every 32-bit n, checked on random and boundary pairs.
static void check_reciprocal_division()
{
    unsigned long long rng = 12345;
    auto next = [&]() {
        rng = rng * 6364136223846793005ull + 1442695040888963407ull;
        return (uint32_t)(rng >> 33);
    };
    for (int it = 0; it < 2000000; ++it) {
        const uint32_t d = (it % 3 == 0) ? (next() % 300 + 1) : (next() % 2000000000u + 1);
        uint32_t n = (it % 5 == 0) ? (next() % (4 * d + 1)) : next() % 2147483647u;
        if (it % 7 == 0 && (n / d) * d + d - 1 > n) n = (n / d) * d + d - 1;  // last value before a multiple
        const unsigned long long mul = d <= 1 ? 0ull : (~0ull / d) + 1ull;
        const uint32_t q = mul == 0 ? n : (uint32_t)(((unsigned __int128)n * mul) >> 64);
        if (q != n / d) {
            ++fails;
            if (fails < 10) std::printf("FAIL reciprocal division n=%u d=%u q=%u\n", n, d, q);
        }
    }
}

int main()
{
    check_reciprocal_division();
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
        {64, 14, 14, 256, 512, 1, 1, 0, 0, 8},  {1, 4, 32, 256, 16, 1, 1, 0, 0, 8},   {1, 4, 32, 2304, 16, 1, 1, 0, 0, 8},
        {1, 6, 6, 256, 32, 3, 3, 1, 1, 8},      {1, 6, 6, 256, 32, 3, 3, 1, 1, 4},    {1, 6, 6, 256, 32, 3, 3, 1, 1, 2},
        {1, 8, 8, 32, 32, 3, 3, 1, 1, 8},       {2, 30, 16, 32, 64, 3, 3, 1, 1, 8},   {1, 16, 24, 32, 48, 5, 5, 2, 2, 8},
        {1, 47, 40, 32, 32, 3, 3, 1, 1, 4},     {1, 47, 40, 64, 32, 3, 3, 1, 1, 2},   {3, 9, 11, 16, 16, 1, 1, 0, 0, 8},
        {2, 32, 32, 3, 32, 5, 5, 2, 2, 8},      {1, 12, 12, 32, 136, 3, 3, 1, 1, 8},  {1, 14, 22, 32, 32, 3, 3, 1, 1, 2},
    };
    for (const auto &v : shapes) check(v[0], v[1], v[2], v[3], v[4], v[5], v[6], v[7], v[8], v[9], 0);
    for (const auto &v : shapes) check(v[0], v[1], v[2], v[3], v[4], v[5], v[6], v[7], v[8], v[9], 1);
    // seeded random shapes across the planner's range (whatever it accepts is checked)
    unsigned long long rng = 0x5EEDC0DEull;
    auto next = [&](int lo, int hi) {  // uniform in [lo, hi]
        rng = rng * 6364136223846793005ull + 1442695040888963407ull;
        return lo + static_cast<int>((rng >> 33) % static_cast<unsigned long long>(hi - lo + 1));
    };
    static const int kBits[4] = {8, 8, 4, 2};
    for (int i = 0; i < 300; ++i) {
        const int bits = kBits[next(0, 3)];
        const int per = 8 / bits;
        const int c = per * next(1, bits == 8 ? 96 : 64);
        const int m = per * next(1, 320 / per);
        const int kh = next(1, 7), kw = next(1, 7);
        const int ph = next(0, kh / 2), pw = next(0, kw / 2);
        const int h = next(std::max(1, kh - 2 * ph), 40), w = next(std::max(1, kw - 2 * pw), 48);
        check(next(1, 3), h, w, c, m, kh, kw, ph, pw, bits, next(0, 1));
    }
    std::printf("fails=%d\n", fails);
    return fails != 0;
}
