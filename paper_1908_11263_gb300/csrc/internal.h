// Host-side interfaces between the C ABI (capi.cu) and the kernel files.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace qnn {

struct ConvShape {
    int n, h, w, c, m, kh, kw, sh, sw, ph, pw, bits, oh, ow;
    int thr;  // staircase compression (thresholds) instead of scaling and clipping
    int pool; // 2x2 stride-2 max-pool of the compressed outputs, fused (strip tiles only)
};

struct ConvParams {
    const uint8_t *x;
    const uint8_t *w;
    const int32_t *bias;    // may be null
    const int16_t *kappa;
    const int32_t *lambda;
    const uint8_t *shifts;  // may be null
    int shift;
    uint8_t *y;
    const int32_t *thresholds;  // [m][2^Q - 1] for staircase compression, else null
};

// ---- INT-1 convolution (XNOR / popcount, CUDA cores) -- conv_binary.cu
cudaError_t launch_conv_binary(const ConvShape &s, const uint8_t *x, const uint8_t *w, const int32_t *thr, uint8_t *y,
                               cudaStream_t st);

// ---- CUDA-core convolution (any stride / padding) -- conv_direct.cu
cudaError_t launch_conv_direct(const ConvShape &s, const ConvParams &p, cudaStream_t st);

// ---- tensor-core implicit GEMM (stride 1) -- conv_tc.cu
struct TcPlan {
    bool ok;
    int nt;             // output channels per tile (MMA N): 16, 32, 64 or 128
    int n_ntiles;       // ceil(m / nt)
    int c_pad;          // channels per tap rounded up to 16
    int cs;             // channels per staged slab
    int nslab;          // c_pad / cs
    int k_pad;          // kh * kw * c_pad
    int rows_max;       // input rows staged per tile (upper bound)
    int p_alloc;        // staged positions per horizontal copy
    int stages;         // converted slabs in flight
    int raw_stages;     // raw input windows in flight
    int b_stages;       // filter tiles in flight (1 when resident)
    int b_resident;     // whole filter set kept in shared memory
    int tiles_per_img;  // row tiles: ceil(oh * ow / 128); strips: ceil(oh / 16) * ceil(ow / 8)
    int strip;          // 16 x 8 strip tiles staged as one padded window (else 128-pixel row tiles)
    int fp8;            // INT-4/INT-2 staged as e4m3 bytes, kind::f8f6f4 MMAs with K = 32 (else fp16, K = 16)
    int sp;             // strips: window width in pixels (8 + kw - 1)
    int ncb;            // strips: column blocks per image
    long long total_tiles;
    int mmas_per_tile;  // MMAs (K = 16 each) per tile
    int limit_mmas;     // most MMAs one exact fp32 accumulator chunk may take
    int chunk_mmas;     // MMAs per exact fp32 accumulator chunk (whole taps)
    int nchunks;        // chunks per tile
    int grp_chunks;     // chunks per accumulator group (one TMEM buffer each, completed together)
    int ngroups;        // accumulator groups in the TMEM ring
    int nsg;            // groups per tile (more than one: running sums kept in TMEM)
    uint32_t row_bytes, raw_bytes, b_bytes, b_tile_bytes, copy_bytes, stage_bytes, smem_bytes, tmem_cols;
    uint32_t off_raw, off_stages, off_chan, off_bar, off_rec;
    size_t workspace_bytes;
};

TcPlan plan_conv_tc(const ConvShape &s);
cudaError_t launch_conv_tc_prep(const TcPlan &plan, const ConvShape &s, const ConvParams &p, void *workspace,
                                cudaStream_t st);
// after_prep: launched right after launch_conv_tc_prep on the same stream, so the
// convolution may start while the preparation kernel still runs.
cudaError_t launch_conv_tc_run(const TcPlan &plan, const ConvShape &s, const uint8_t *x, uint8_t *y,
                               const void *workspace, cudaStream_t st, bool after_prep);

// ---- tensor-core window kernel (stride 1, one launch per layer) -- conv_win*.cu
// Tiles of S strips (16 output rows x 8 columns each) staged as one padded
// window; filters re-laid out and per-channel constants derived in shared
// memory by the kernel itself; exact-chunk count derived from the filters.
struct WinPlan {
    bool ok;
    int nt;               // MMA N: all output channels, rounded up to 32, 64 or 128
    int fp8;              // e4m3 staging, kind::f8f6f4 (INT-4/INT-2), else fp16, kind::f16 (INT-8)
    int kch;              // channels per 16-byte K-chunk: 8 (fp16) or 16 (e4m3)
    int c_pad;            // channels per tap rounded up to two K-chunks
    int groups;           // K-chunks per tap (c_pad / kch)
    int fold;             // kernel columns folded into K (INT-8, C not a multiple of 8, C * kw <= 16, m <= 64):
                          // a staged position holds its kw horizontal neighbours' channels, one MMA "tap"
                          // per kernel row
    int kwf;              // kernel columns as the MMAs see them: kw, or 1 when folded
    int taps;             // kh * kw, or kh when folded
    int ksteps;           // MMAs per tap (groups / 2)
    int s;                // strips per tile (1 or 2)
    int sp, wh;           // window width and height in pixels
    int p_alloc;          // staged positions per K-chunk plane
    int tiles_x, tiles_y, tiles_per_img;
    long long total_tiles;
    int full_rows;        // a window spans whole image rows: one bulk copy per tile
    int nch_max;          // exact fp32 chunks the worst-case filters would need
    int nch_min;          // fewest chunks per strip the kernel considers (1)
    int raw_stages, a_stages;
    uint32_t raw_row_bytes, raw_bytes, b_bytes, chunk_stride, stage_bytes;
    uint32_t off_b, off_a, off_raw, off_rec, off_thr, off_tap, off_mtab, off_pre, off_wraw, off_bar, smem_bytes;
    uint32_t wraw_bytes;  // packed filters bulk-copied into shared memory (0: read from global memory)
    uint32_t tail_bytes;  // shared memory from off_rec to the end of the pre-load operands
    size_t img_bytes;     // qconv_hwc_prepare workspace: the prepared image (B, then the tail)
};

WinPlan plan_conv_win(const ConvShape &s);
// One launch of the window kernel.  With img == nullptr it prepares the
// caller's filters and constants (p.w, p.bias, ...) itself; with img it reads
// the image qconv_hwc_prepare wrote (img_bytes at img) and p carries only x, y.
cudaError_t launch_conv_win(const WinPlan &plan, const ConvShape &s, const ConvParams &p, cudaStream_t st,
                            const void *img = nullptr);
// qconv_hwc_prepare for the window kernel: one block prepares the filters and
// constants exactly as a convolving launch would and writes the image
// (plan.img_bytes) to `workspace`.
cudaError_t prepare_conv_win(const WinPlan &plan, const ConvShape &s, const ConvParams &p, void *workspace,
                             cudaStream_t st);

// ---- max-pool, fully connected, packing
cudaError_t launch_maxpool(int n, int h, int w, int c, int k, int s, int bits, const uint8_t *x, uint8_t *y,
                           cudaStream_t st);
cudaError_t launch_linear(int n, int k, int m, const uint8_t *x, const int8_t *w, const int32_t *bias, int32_t *y,
                          cudaStream_t st);
cudaError_t launch_pack(const int8_t *src, uint8_t *dst, long long count, int bits, cudaStream_t st);
cudaError_t launch_unpack(const uint8_t *src, int8_t *dst, long long count, int bits, int is_signed,
                          cudaStream_t st);

// number of SMs of the current device (cached per device)
int device_sm_count();

// device address of the library's status word on the current device (cached per device; null on failure)
int *device_status_ptr();

}  // namespace qnn
