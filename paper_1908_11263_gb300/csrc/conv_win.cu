// Host side of the window kernel (conv_win.cuh): the planner, the launches
// (convolving, and the one-block launch that writes a prepared image) and the
// prepared-workspace layout.
#include <algorithm>

#include "conv_win.cuh"

namespace qnn {

namespace {

uint32_t round_up(uint32_t v, uint32_t a) { return (v + a - 1) / a * a; }
size_t round_up_sz(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Shared-memory bytes of the barriers and the words after them (see the kernel).
constexpr uint32_t kBarBytes = (4 * win::kMaxStages + 2 * win::kMaxSlots + 3) * 8 + sizeof(win::Misc);

// Strips per tile: two unless the image is at most 8 columns wide, or the
// second strip of a tile would compute more than 15 % extra columns.
int strips_per_tile(int ow)
{
    if (ow <= win::kCols) return 1;
    const long long w1 = (ow + 7) / 8 * 8LL, w2 = (ow + 15) / 16 * 16LL;
    return w2 * 100 <= w1 * 115 ? 2 : 1;
}

}  // namespace

WinPlan plan_conv_win(const ConvShape &s)
{
    WinPlan p{};
    p.ok = false;
    if (s.sh != 1 || s.sw != 1 || s.oh <= 0 || s.ow <= 0 || s.n < 0) return p;
    p.fp8 = s.bits != 8;
    p.kch = p.fp8 ? 16 : 8;
    // INT-8 with few channels (C * kw <= 16, C not a multiple of 8): a kernel row's kw * C
    // values of a position fill one 16-value K-step (two K-chunks)
    p.fold = s.bits == 8 && s.c % 8 != 0 && s.kw > 1 && s.c * s.kw <= 16 && s.m <= 64;
    p.kwf = p.fold ? 1 : s.kw;
    // INT-8 in fp16 (whole 8-channel chunks), INT-4 / INT-2 in e4m3 (whole 32-channel pairs)
    if (!p.fold && (s.bits == 8 ? (s.c % 8 != 0) : (s.c % 32 != 0))) return p;
    if (s.m > 128) return p;  // one filter set, all output channels in one MMA N
    p.nt = s.m <= 32 ? 32 : s.m <= 64 ? 64 : 128;
    // staged values per position and "tap" (a tap is a kernel row when folded)
    p.c_pad = p.fold ? 16 : (s.c + 2 * p.kch - 1) / (2 * p.kch) * (2 * p.kch);
    p.groups = p.c_pad / p.kch;
    if (p.groups > 8) return p;  // the window holds every channel of a pixel
    p.taps = p.fold ? s.kh : s.kh * s.kw;
    if (s.kh > 8 || s.kw > 8 || p.taps > win::kMaxTaps) return p;
    p.ksteps = p.groups / 2;
    const long long cb = static_cast<long long>(s.c) * s.bits / 8;
    // worst-case exact chunks: products of at most max|staged x| * max|w| each,
    // whole taps (c_pad products per accumulator per tap) per chunk
    const long long max_prod = p.fp8 ? (s.bits == 4 ? 15 * 8 : 3 * 2) : 128 * 128;
    const long long taps_per_chunk = ((1ll << 22) / max_prod) / p.c_pad;
    if (taps_per_chunk < 1) return p;
    p.nch_max = static_cast<int>((p.taps + taps_per_chunk - 1) / taps_per_chunk);
    if (p.nch_max > 16) return p;
    const int s_pref = strips_per_tile(s.ow);
    for (int S : {s_pref, 3 - s_pref}) {
        // the kernel takes the fewest chunks the filters allow (MMAs that accumulate
        // into one TMEM buffer issue back to back at the full rate)
        const int nmin = 1;
        if (S * std::max(nmin, p.nch_max) * p.nt > 512) continue;  // one slot of accumulators in TMEM
        // folded positions carry their kw - 1 right neighbours: no extra window columns
        const int sp = win::kCols * S + (p.fold ? 0 : s.kw - 1), wh = win::kRows + s.kh - 1;
        if (wh * sp > win::kMaxKP * 128) continue;  // converter positions per thread
        const int tiles_x = (s.ow + win::kCols * S - 1) / (win::kCols * S);
        const bool full_rows = tiles_x == 1 || p.fold;  // folded windows read whole rows
        const long long row_bytes = s.w * cb;
        uint32_t raw_row_bytes;
        if (full_rows) {
            if (row_bytes % 16 != 0 || row_bytes > (1 << 20)) continue;  // rows move as one bulk copy
            raw_row_bytes = static_cast<uint32_t>(row_bytes);
        } else {
            if (cb % 16 != 0) continue;  // per-row copies start at any pixel
            raw_row_bytes = round_up(static_cast<uint32_t>(std::min(sp, s.w) * cb), 16);
        }
        const uint32_t raw_bytes = round_up(static_cast<uint32_t>(std::min(wh, s.h)) * raw_row_bytes, 128);
        if (raw_bytes >= (1u << 20)) continue;  // one transaction count
        const uint32_t p_alloc = round_up(static_cast<uint32_t>(wh * sp), 8);
        const uint32_t chunk_stride = p_alloc * 16;
        const uint32_t stage_bytes = chunk_stride * p.groups;
        const uint32_t b_bytes = static_cast<uint32_t>(p.taps * p.groups * p.nt * 16);
        // rec0, rec1 (16 bytes each), direct flags (1 per 16 channels)
        const uint32_t rec_bytes = round_up(static_cast<uint32_t>(2 * p.nt * 16 + p.nt / 16), 16);
        const uint32_t thr_bytes = s.thr ? static_cast<uint32_t>(p.nt * kThrStride * 4) : 0u;
        const uint32_t tap_bytes = round_up(static_cast<uint32_t>((p.taps + 3) * p.nt * 4), 16);
        const uint32_t mtab_bytes = round_up(static_cast<uint32_t>(S * p.taps * p.ksteps * 8), 16);
        const uint32_t pre_bytes = 4096u + static_cast<uint32_t>(p.nt) * 32u;  // pre-load MMA operands
        // the packed filters are bulk-copied into shared memory when they are whole 16-byte units and fit
        const long long wraw = static_cast<long long>(s.m) * s.kh * s.kw * cb;
        bool placed = false;
        for (int copy_w : {1, 0}) {
          if (copy_w && (wraw % 16 != 0 || wraw > 96 * 1024)) continue;
          const uint32_t wraw_bytes = copy_w ? static_cast<uint32_t>(wraw) : 0u;
          for (int as : {3, 2}) {
            for (int rs : {3, 2}) {
                uint32_t off = 0;
                const uint32_t off_b = off;
                off = round_up(off + b_bytes, 128);
                const uint32_t off_a = off;
                off = round_up(off + as * stage_bytes, 128);
                const uint32_t off_raw = off;
                off = round_up(off + rs * raw_bytes, 128);
                const uint32_t off_rec = off;
                off += rec_bytes;
                const uint32_t off_thr = off;
                off += thr_bytes;
                const uint32_t off_tap = off;
                off += tap_bytes;
                const uint32_t off_mtab = round_up(off, 16);
                off = off_mtab + mtab_bytes;
                const uint32_t off_pre = round_up(off, 128);
                off = off_pre + pre_bytes;
                const uint32_t off_wraw = round_up(off, 128);
                off = off_wraw + wraw_bytes;
                const uint32_t off_bar = round_up(off, 16);
                const uint32_t total = off_bar + kBarBytes;
                // descriptor start addresses are 14-bit fields of 16-byte units (256 KB)
                if (total > static_cast<uint32_t>(win::kSmemLimit)) continue;
                p.off_mtab = off_mtab;
                p.off_pre = off_pre;
                p.off_wraw = off_wraw;
                p.wraw_bytes = wraw_bytes;
                p.a_stages = as;
                p.raw_stages = rs;
                p.off_b = off_b;
                p.off_a = off_a;
                p.off_raw = off_raw;
                p.off_rec = off_rec;
                p.off_thr = off_thr;
                p.off_tap = off_tap;
                p.off_bar = off_bar;
                p.smem_bytes = total;
                placed = true;
                break;
            }
            if (placed) break;
          }
          if (placed) break;
        }
        if (!placed) continue;
        p.s = S;
        p.nch_min = nmin;
        p.sp = sp;
        p.wh = wh;
        p.p_alloc = static_cast<int>(p_alloc);
        p.tiles_x = tiles_x;
        p.tiles_y = (s.oh + win::kRows - 1) / win::kRows;
        p.tiles_per_img = p.tiles_x * p.tiles_y;
        p.total_tiles = static_cast<long long>(s.n) * p.tiles_per_img;
        if (p.total_tiles >= (1ll << 31)) return p;
        p.full_rows = full_rows;
        p.raw_row_bytes = raw_row_bytes;
        p.raw_bytes = raw_bytes;
        p.b_bytes = b_bytes;
        p.chunk_stride = chunk_stride;
        p.stage_bytes = stage_bytes;
        // prepared workspace: the image of B and the tail
        p.tail_bytes = p.off_pre + 4096u + static_cast<uint32_t>(p.nt) * 32u - p.off_rec;
        p.img_bytes = round_up_sz(static_cast<size_t>(b_bytes) + p.tail_bytes, 256);
        p.ok = true;
        return p;
    }
    return p;
}

namespace {

win::WinArgs win_args(const WinPlan &plan, const ConvShape &s, const ConvParams &p)
{
    win::WinArgs a{};
    a.x = p.x;
    a.y = p.y;
    a.w = p.w;
    a.bias = p.bias;
    a.kappa = p.kappa;
    a.lambda = p.lambda;
    a.shifts = p.shifts;
    a.thr = s.thr ? p.thresholds : nullptr;
    a.shift = p.shift;
    a.n = s.n; a.h = s.h; a.w_ = s.w; a.c = s.c; a.m = s.m; a.kh = s.kh; a.kw = s.kw;
    a.ph = s.ph; a.pw = s.pw; a.oh = s.oh; a.ow = s.ow;
    a.c_pad = plan.c_pad;
    a.groups = plan.groups;
    a.taps = plan.taps;
    a.fold = plan.fold;
    a.kwf = plan.kwf;
    a.ksteps = plan.ksteps;
    a.s = plan.s;
    a.sp = plan.sp;
    a.wh = plan.wh;
    a.npos = plan.wh * plan.sp;
    a.cb = s.c * s.bits / 8;
    a.full_rows = plan.full_rows;
    a.tiles_x = plan.tiles_x;
    a.tiles_per_img = plan.tiles_per_img;
    a.total_tiles = static_cast<int>(plan.total_tiles);
    a.fd_tpi = make_fastdiv(static_cast<uint32_t>(plan.tiles_per_img));
    a.fd_tx = make_fastdiv(static_cast<uint32_t>(plan.tiles_x));
    a.fd_sp = make_fastdiv(static_cast<uint32_t>(plan.sp));
    a.raw_stages = plan.raw_stages;
    a.a_stages = plan.a_stages;
    a.nch_max = plan.nch_max;
    a.nch_min = plan.nch_min;
    a.raw_row_bytes = plan.raw_row_bytes;
    a.raw_bytes = plan.raw_bytes;
    a.chunk_stride = plan.chunk_stride;
    a.stage_bytes = plan.stage_bytes;
    a.off_b = plan.off_b;
    a.off_a = plan.off_a;
    a.off_raw = plan.off_raw;
    a.off_rec = plan.off_rec;
    a.off_thr = plan.off_thr;
    a.off_tap = plan.off_tap;
    a.off_bar = plan.off_bar;
    a.off_mtab = plan.off_mtab;
    a.off_pre = plan.off_pre;
    a.off_wraw = plan.off_wraw;
    a.wraw_bytes = plan.wraw_bytes;
    a.pool = s.pool;
    a.pool_oh = s.oh / 2;
    a.pool_ow = s.ow / 2;
    a.b_bytes = plan.b_bytes;
    a.tail_bytes = plan.tail_bytes;
    a.status = device_status_ptr();
    return a;
}

cudaError_t launch_win(const WinPlan &plan, const ConvShape &s, const win::WinArgs &a, int grid, cudaStream_t st)
{
    if (!a.status) return cudaErrorInvalidSymbol;
    switch (s.bits) {
        case 8: return launch_win_bits<8>(a, plan.nt, grid, plan.smem_bytes, st);
        case 4: return launch_win_bits<4>(a, plan.nt, grid, plan.smem_bytes, st);
        default: return launch_win_bits<2>(a, plan.nt, grid, plan.smem_bytes, st);
    }
}

}  // namespace

cudaError_t launch_conv_win(const WinPlan &plan, const ConvShape &s, const ConvParams &p, cudaStream_t st,
                            const void *img)
{
    if (s.n == 0) return cudaSuccess;
    win::WinArgs a = win_args(plan, s, p);
    if (img) {
        a.img = static_cast<const uint8_t *>(img);
        a.wraw_bytes = 0;  // no filter copy: the image replaces it
    }
    const long long sms = device_sm_count();
    const int grid = static_cast<int>(std::min<long long>(plan.total_tiles, sms));
    return launch_win(plan, s, a, grid, st);
}

cudaError_t prepare_conv_win(const WinPlan &plan, const ConvShape &s, const ConvParams &p, void *workspace,
                             cudaStream_t st)
{
    win::WinArgs a = win_args(plan, s, p);
    a.img_out = static_cast<uint8_t *>(workspace);
    return launch_win(plan, s, a, 1, st);
}

}  // namespace qnn
