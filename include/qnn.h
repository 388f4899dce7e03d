/*
 * qnn.h - C ABI of the GB300 (sm_103a) quantized HWC convolution library.
 *
 * Method: PULP-NN, "Accelerating Quantized Neural Networks on Parallel
 * Ultra-Low-Power RISC-V Processors" (arXiv 1908.11263).  The library runs the
 * data-parallel hot path of that method on one GPU: im2col + integer MatMul
 * with 32-bit accumulation (Sec. III-B, Eq. 2 and Eq. 6), compression of the
 * accumulator back to Q bits (Sec. III-A), max-pooling and the fully connected
 * layer (Sec. IV-A), for INT-8 and packed INT-4 / INT-2 data (Sec. IV-A,
 * "Sub-byte Extensions").  Also: the staircase (threshold) compression of
 * Eq. 4, the INT-1 XNOR / popcount convolution of Eq. 5, and a convolution
 * with its 2x2 max-pooling fused into one kernel.
 *
 * Conventions shared by every entry point
 *  - Plain C types only.  Pointers marked "device" must point to memory of the
 *    current CUDA device; the caller allocates and owns every buffer, and keeps
 *    it alive until the work queued on `stream` has finished.
 *  - `stream` is a cudaStream_t passed as void*; NULL means the legacy default
 *    stream.  Every call only enqueues work and returns; device-side problems
 *    surface at the caller's next synchronisation, or through
 *    qnn_device_status().
 *  - Arguments are validated before anything is launched; a call that returns
 *    an error has enqueued nothing.  Nothing is thrown across the ABI.
 *  - Tensors are dense and contiguous; there are no stride arguments.  Input
 *    and output buffers must not overlap.
 *  - Sub-byte storage: element e of a packed Q-bit stream sits in byte
 *    e / (8/Q) at bits [(e mod (8/Q)) * Q, +Q), the first element in the least
 *    significant bits.  Activations are unsigned, weights two's-complement.
 *  - Thread safety: calls may be made from several host threads; the only
 *    shared host state is a per-device cache of queried device properties.
 */
#ifndef QNN_H
#define QNN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    QNN_OK = 0,
    QNN_EINVAL = 1,        /* NULL pointer, non-positive size, empty output, shift out of [0,62], bad struct_size */
    QNN_EUNSUPPORTED = 2,  /* bits not in {8,4,2}; mixed bit-widths; C, M or a count not a whole number of bytes
                              at Q bits; accumulator bound above int32; forced algorithm that cannot run the shape */
    QNN_EALIGN = 3,        /* a tensor pointer that must be 16-byte aligned is not */
    QNN_ECUDA = 4,         /* a CUDA runtime call or kernel launch failed */
    QNN_ETIMEOUT = 5,      /* a bounded device-side wait gave up (reported by qnn_device_status) */
    QNN_EWORKSPACE = 6,    /* workspace missing or smaller than qconv_hwc_workspace_size() */
    QNN_ESCRATCH = 7       /* qconv_hwc_noalloc(): the layer needs more than QNN_NOALLOC_SCRATCH_BYTES */
} qnn_status;

/* Convolution algorithm choice (qnn_conv_desc.algo). */
enum {
    QNN_ALGO_AUTO = 0,         /* tensor-core kernel when the shape allows it, else the CUDA-core kernel */
    QNN_ALGO_DIRECT = 1,       /* CUDA-core kernel (dp4a), any stride / padding */
    QNN_ALGO_TENSORCORE = 2,   /* tcgen05 implicit GEMM (the window kernel when its plan fits, else the
                                  general one); QNN_EUNSUPPORTED when neither fits the shape */
    QNN_ALGO_TC_WINDOW = 3,    /* the window kernel only: stride 1, m <= 128, INT-8 with c a multiple of 8
                                  or INT-4/INT-2 with c a multiple of 32, c <= 64 (INT-8) or 128 (sub-byte),
                                  kh, kw <= 8; one launch per call, filters read in place */
    QNN_ALGO_TC_GENERAL = 4    /* the general tensor-core kernel only (filter preparation kernel plus
                                  convolution kernel, any stride-1 shape with whole 16-byte input rows) */
};

/*
 * One convolution layer (Sec. III-B).  Input x is NHWC [n][h][w][c]; filters
 * are [m][kh][kw][c] with c innermost, so each bank W(m) is stored in im2col
 * order (Eq. 6).  Output y is NHWC [n][oh][ow][m] with
 * oh = (h + 2*pad_h - kh) / stride_h + 1 and ow likewise (floor).  Padding
 * reads as activation 0.  x, w and y all use `bits` per element.
 */
typedef struct {
    uint32_t struct_size;      /* = sizeof(qnn_conv_desc) */
    int32_t n, h, w, c;        /* input batch, height, width, channels; n may be 0 (no work) */
    int32_t m, kh, kw;         /* output channels, kernel height and width */
    int32_t stride_h, stride_w;
    int32_t pad_h, pad_w;
    int32_t bits;              /* Q in {8, 4, 2} for activations, weights and outputs alike */
    int32_t shift;             /* right shift in [0, 62], used for every channel when shifts == NULL */
    int32_t algo;              /* QNN_ALGO_* */
} qnn_conv_desc;

/*
 * Bytes of device workspace for this layer: what qconv_hwc_prepare() writes
 * and qconv_hwc_run() reads, and what qconv_hwc() needs on the general
 * tensor-core kernel (0 for the CUDA-core kernel).  For the general kernel
 * the workspace holds the filters re-laid out for the tensor cores and the
 * per-channel compression constants, rewritten by every qconv_hwc() call, so
 * one workspace must not be shared by calls that can run concurrently.  For
 * the window kernel it holds the image of the kernel's shared-memory operands
 * that qconv_hwc_prepare() builds once (the filters as the tensor-core B
 * operand, the per-channel compression records, the exact chunk count and the
 * MMA issue table); qconv_hwc_run() reads it with two bulk copies per block,
 * and qconv_hwc() builds the same operands inside its one launch and leaves
 * the workspace alone.
 */
qnn_status qconv_hwc_workspace_size(const qnn_conv_desc *d, size_t *bytes);

/*
 * Quantized convolution with fused compression (Sec. III-A, III-B, IV-A):
 *
 *   acc[n][oy][ox][o] = sum_{i<kh, j<kw, ch<c} x[n][oy*sh-ph+i][ox*sw-pw+j][ch] * w[o][i][j][ch]   (int32)
 *   y[n][oy][ox][o]   = clip( floor( ((acc + bias[o]) * kappa[o] + lambda[o]) / 2^shift_o ), 0, 2^Q - 1 )
 *
 * computed exactly (64-bit intermediate for the scaled value); the clip is
 * also the ReLU.  shift_o = shifts[o] when shifts != NULL, else d->shift.
 *
 *   x       device, packed unsigned Q-bit NHWC, 16-byte aligned
 *   w       device, packed signed Q-bit [m][kh][kw][c], 16-byte aligned
 *   bias    device int32[m], or NULL for zero
 *   kappa   device int16[m]
 *   lambda  device int32[m]
 *   shifts  device uint8[m] with values in [0, 62], or NULL
 *   y       device, packed unsigned Q-bit NHWC output, 16-byte aligned
 *   workspace, workspace_bytes: device scratch of at least
 *           qconv_hwc_workspace_size() bytes, 256-byte aligned (may be NULL
 *           when that size is 0).  When the window kernel serves the layer
 *           (qconv_hwc_tc_kernel() == QNN_ALGO_TC_WINDOW) the call is one
 *           launch that reads w, bias, kappa, lambda and shifts in place and
 *           the workspace is neither read nor written (it may be NULL).
 *
 * Requirements (else QNN_EUNSUPPORTED): c and m multiples of 8/Q, and
 * kh*kw*c*(2^Q-1)*2^(Q-1) < 2^30, so that the int32 accumulator of Eq. 2 cannot
 * overflow.  The caller keeps |bias| < 2^30 (bias values are not inspected).
 */
qnn_status qconv_hwc(const qnn_conv_desc *d, const void *x, const void *w, const int32_t *bias,
                     const int16_t *kappa, const int32_t *lambda, const uint8_t *shifts, void *y,
                     void *workspace, size_t workspace_bytes, void *stream);

/*
 * The two halves of qconv_hwc(), for callers whose filters and compression
 * constants stay fixed across many calls (inference serving):
 *
 * qconv_hwc_prepare: writes into `workspace` the filters re-laid out for the
 *   tensor cores and the per-channel constants derived from bias, kappa,
 *   lambda and the shifts (same argument rules as qconv_hwc); one small
 *   launch.  The caller's buffers may be freed or changed afterwards.  For a
 *   descriptor that selects the CUDA-core kernel it enqueues nothing.
 * qconv_hwc_run: the convolution itself, reading a workspace prepared for the
 *   same descriptor (any other workspace content gives undefined results).
 *   Only for descriptors that select the tensor-core kernel; otherwise
 *   QNN_EUNSUPPORTED.  The window kernel launches with programmatic stream
 *   serialization: it may start while the previous kernel in the stream is
 *   still running, waits for it before touching x or y, and reads the
 *   workspace before that wait, so the workspace must not be written by the
 *   kernel launched just before it (qconv_hwc_prepare's own launch is fine:
 *   its successor starts only after it ends).
 * qconv_hwc(...) is exactly qconv_hwc_prepare(...) followed by qconv_hwc_run(...)
 * on the same stream.
 */
qnn_status qconv_hwc_prepare(const qnn_conv_desc *d, const void *w, const int32_t *bias, const int16_t *kappa,
                             const int32_t *lambda, const uint8_t *shifts, void *workspace, size_t workspace_bytes,
                             void *stream);
qnn_status qconv_hwc_run(const qnn_conv_desc *d, const void *x, void *y, const void *workspace,
                         size_t workspace_bytes, void *stream);

/*
 * Quantized convolution, compression and 2x2 max-pooling in one kernel: the
 * pooling layer of Sec. IV-A (window 2, stride 2, no padding, floor output
 * size) applied to the output of qconv_hwc(), fused into its epilogue so the
 * full-resolution output never reaches memory:
 *
 *   t[n][oy][ox][o]  = y of qconv_hwc() for the same arguments
 *   y[n][py][px][o]  = max over dy, dx in {0, 1} of t[n][2*py+dy][2*px+dx][o]
 *                      for py < oh / 2, px < ow / 2 (integer division)
 *
 * Arguments are those of qconv_hwc(); y is the pooled NHWC tensor
 * [n][oh/2][ow/2][m], packed Q-bit, 16-byte aligned.  The workspace size is
 * qconv_hwc_workspace_size() of the same descriptor.  Runs only on the
 * tensor-core kernel (stride 1, the shapes qconv_hwc_algo() reports as
 * QNN_ALGO_TENSORCORE, d->algo not QNN_ALGO_DIRECT); QNN_EUNSUPPORTED
 * otherwise, and QNN_EINVAL when oh or ow is below 2 (no pooled pixel).
 */
qnn_status qconv_hwc_pool2(const qnn_conv_desc *d, const void *x, const void *w, const int32_t *bias,
                           const int16_t *kappa, const int32_t *lambda, const uint8_t *shifts, void *y,
                           void *workspace, size_t workspace_bytes, void *stream);

/*
 * qconv_hwc_pool2_run: qconv_hwc_pool2() on filters prepared with
 * qconv_hwc_prepare() for the same descriptor: the fused convolution,
 * compression and 2x2/2 max-pool, one launch that reads x, the workspace and
 * writes the pooled y ([n][oh/2][ow/2][m], packed Q-bit, 16-byte aligned).
 * Only where qconv_hwc_algo() reports the window tensor-core kernel
 * (qconv_hwc_tc_kernel() == QNN_ALGO_TC_WINDOW); QNN_EUNSUPPORTED otherwise,
 * QNN_EINVAL when oh or ow is below 2, QNN_EWORKSPACE for a workspace below
 * qconv_hwc_workspace_size() or not 256-byte aligned.  The workspace rules of
 * qconv_hwc_run() apply (it is read before the wait on the previous kernel).
 */
qnn_status qconv_hwc_pool2_run(const qnn_conv_desc *d, const void *x, void *y, const void *workspace,
                               size_t workspace_bytes, void *stream);

/*
 * Quantized convolution with staircase compression (Sec. III-A, Eq. 4), the
 * paper's compression for INT-4 and INT-2 outputs:
 *
 *   acc[n][oy][ox][o] = as in qconv_hwc() (int32, no bias)
 *   y[n][oy][ox][o]   = number of k in [0, 2^Q - 1) with thresholds[o][k] <= acc
 *
 * For thresholds sorted ascending per channel this is the index p of the
 * interval [tau_p, tau_p+1) that holds the accumulator, counted from 0 for the
 * lowest interval (unsigned outputs).  The thresholds absorb bias and batch
 * normalisation (footnote to Eq. 3), so there is no bias, kappa or lambda.
 *
 *   x, w, y     as in qconv_hwc(); d->bits must be 4 or 2 (else QNN_EUNSUPPORTED)
 *   thresholds  device int32 [m][2^Q - 1], 4-byte aligned (any values)
 *   workspace, workspace_bytes: as in qconv_hwc() (qconv_hwc_workspace_size)
 *
 * d->shift is ignored.  Same accumulator bound and other requirements as
 * qconv_hwc().
 */
qnn_status qconv_hwc_thresholds(const qnn_conv_desc *d, const void *x, const void *w, const int32_t *thresholds,
                                void *y, void *workspace, size_t workspace_bytes, void *stream);

/*
 * INT-1 convolution (Sec. III-A, Eq. 5; binary kernel of Sec. IV-A).  Values
 * +1 / -1 are bits 1 / 0, eight per byte, element e at bit e mod 8 of byte e / 8
 * (the sub-byte order above with Q = 1).
 *
 *   acc[n][oy][ox][o] = number of (i, j, ch) with the input pixel inside the
 *                       image and bit(w[o][i][j][ch]) == bit(x[n][iy][ix][ch])
 *                       (popcount of W xnor X; padding contributes nothing)
 *   y[n][oy][ox][o]   = 1 if thresholds[o] <= acc, else 0
 *
 *   d           d->bits must be 1; c and m multiples of 8; d->shift and d->algo ignored
 *   x           device, NHWC bits [n][h][w][c / 8 bytes]
 *   w           device, [m][kh][kw][c / 8 bytes]
 *   thresholds  device int32 [m], 4-byte aligned
 *   y           device, NHWC bits [n][oh][ow][m / 8 bytes]
 *
 * Runs on CUDA cores (XNOR and population count).  QNN_EUNSUPPORTED when bits
 * is not 1 or c, m are not multiples of 8.
 */
qnn_status qconv_hwc_binary(const qnn_conv_desc *d, const void *x, const void *w, const int32_t *thresholds,
                            void *y, void *stream);

/* Which kernel qconv_hwc() would run for d: QNN_ALGO_DIRECT or QNN_ALGO_TENSORCORE;
 * negative qnn_status on invalid or unsupported descriptors. */
int32_t qconv_hwc_algo(const qnn_conv_desc *d);

/* Which tensor-core kernel qconv_hwc() would run for d: QNN_ALGO_TC_WINDOW or
 * QNN_ALGO_TC_GENERAL; 0 when d selects the CUDA-core kernel; negative qnn_status
 * on invalid or unsupported descriptors. */
int32_t qconv_hwc_tc_kernel(const qnn_conv_desc *d);

/* Operand format of the tensor-core MMAs qconv_hwc() would issue for d, so that a
 * caller can take the right tensor roof: 16 for fp16 operands (tcgen05 kind::f16,
 * the exact embedding of INT-8 and of sub-byte layers with c not a multiple of 32),
 * 8 for e4m3 operands (kind::f8f6f4, twice the fp16 rate per MMA; INT-4/INT-2 with
 * c a multiple of 32), 0 when d selects the CUDA-core kernel; negative qnn_status
 * on invalid or unsupported descriptors.  Not a paper concept: a query about this
 * library's kernel choice. */
int32_t qconv_hwc_mma_operand_bits(const qnn_conv_desc *d);

/* Size of the fixed scratch array behind qconv_hwc_noalloc(): 2 MiB. */
enum { QNN_NOALLOC_SCRATCH_BYTES = 2097152 };

/*
 * qconv_hwc() without a workspace, for callers that cannot allocate device
 * memory.  The paper has no counterpart to this entry point; it serves users of
 * the library.  Typical such callers: a serving runtime that commits all device
 * memory to its own arenas up front and has none to hand to a library; a
 * latency-critical loop, where cudaMalloc / cudaFree would synchronise the
 * device and stall its other streams; a plain C caller with no device
 * allocator of its own to size, own and free a workspace.
 *
 * Arguments and results are those of qconv_hwc() minus the workspace.  The
 * re-laid-out filters and per-channel constants go to one scratch array of
 * QNN_NOALLOC_SCRATCH_BYTES compiled into the library's device image, which
 * every GPU that loads the library holds until the process exits.  The call
 * allocates nothing: no cudaMalloc, cudaFree or allocating library routine.
 *
 *  - Only for descriptors that select the tensor-core kernel (QNN_ALGO_AUTO
 *    resolving to it, or QNN_ALGO_TENSORCORE), else QNN_EUNSUPPORTED.  The
 *    CUDA-core kernel needs no scratch: call qconv_hwc() with a NULL workspace.
 *  - QNN_ESCRATCH, with nothing enqueued, when the layer needs more than
 *    QNN_NOALLOC_SCRATCH_BYTES; qconv_hwc_workspace_size() gives the need.
 *  - Set-up on first use: the first call on each device looks up the scratch
 *    array's device address (cudaGetSymbolAddress, with that device current;
 *    QNN_ECUDA if that fails), and the first tensor-core launch of each bit
 *    width and filter tile on a device raises that kernel's shared-memory
 *    limit.  Make those first calls before any stream capture.
 *  - Shared state: all calls on a device use the same array, which keeps the
 *    last call's contents.  Each call rewrites every scratch byte its
 *    convolution reads before reading it, so nothing has to be cleared between
 *    calls.  Calls that overlap on the GPU (streams with no ordering between
 *    them) race on the array and give undefined results; calls queued on one
 *    stream do not overlap.
 *  - n == 0: after validation, returns QNN_OK with nothing enqueued (the
 *    scratch array is not touched).
 */
qnn_status qconv_hwc_noalloc(const qnn_conv_desc *d, const void *x, const void *w, const int32_t *bias,
                             const int16_t *kappa, const int32_t *lambda, const uint8_t *shifts, void *y,
                             void *stream);

/*
 * Fully connected layer (Sec. IV-A, matrix-vector product split over output
 * neurons in Sec. IV-B), without compression:
 *   y[b][o] = sum_{i<k} x[b][i] * w[o][i] + bias[o]      (int32 output)
 *   x    device uint8 [n][k]      (HWC-flattened activations)
 *   w    device int8  [m][k]
 *   bias device int32 [m] or NULL
 *   y    device int32 [n][m]
 * Requirements: k * 255 * 128 < 2^30 (else QNN_EUNSUPPORTED); the caller keeps |bias| < 2^30.
 */
qnn_status qlinear(int32_t n, int32_t k, int32_t m, const uint8_t *x, const int8_t *w, const int32_t *bias,
                   int32_t *y, void *stream);

/*
 * Max-pooling (Sec. IV-A): y[b][oy][ox][ch] = max_{i,j<k} x[b][oy*s+i][ox*s+j][ch]
 * on packed unsigned Q-bit NHWC data, no padding, oh = (h-k)/s + 1 (floor).
 *   x  device, [n][h][w][c] packed at `bits`;  y  device, [n][oh][ow][c] packed at `bits`
 * Requirements: c a multiple of 8/Q; 1 <= k <= min(h, w); s >= 1.
 */
qnn_status qmaxpool(int32_t n, int32_t h, int32_t w, int32_t c, int32_t k, int32_t s, int32_t bits,
                    const void *x, void *y, void *stream);

/*
 * Sub-byte packing (Sec. IV-A, "Sub-byte Extensions": two INT-4 or four INT-2
 * values per byte, and the unpack-to-INT-8 helper of the same section).
 *   pack_subbyte:   src device int8[count] (the low Q bits of each value are stored),
 *                   dst device uint8[count*Q/8]
 *   unpack_subbyte: src device uint8[count*Q/8], dst device int8[count];
 *                   is_signed != 0 sign-extends (weights), 0 zero-extends (activations)
 * count must be a multiple of 8/Q; bits in {8,4,2} (8 is a plain copy).
 */
qnn_status pack_subbyte(const int8_t *src, void *dst, int64_t count, int32_t bits, void *stream);
qnn_status unpack_subbyte(const void *src, int8_t *dst, int64_t count, int32_t bits, int32_t is_signed,
                          void *stream);

/*
 * Synchronises `stream`, then returns and clears the library's device status
 * word: QNN_OK, or QNN_ETIMEOUT when a bounded wait inside a kernel gave up
 * (the kernel then skipped its remaining work and returned).  QNN_ECUDA when
 * the synchronisation itself fails.
 */
qnn_status qnn_device_status(void *stream);

/*
 * Diagnostics: runs the library's bounded-wait failure path on the GPU.  One
 * warp waits on an mbarrier that nothing arrives on; after `limit_cycles` SM
 * cycles the wait gives up, records QNN_ETIMEOUT in the device status word and
 * the kernel returns, leaving the context usable.  Every wait inside the
 * library's kernels is bounded the same way (a wait that never completes
 * turns into QNN_ETIMEOUT, not a hang).  The paper has no counterpart; this
 * exists so that the failure path can be tested without faulting a GPU.
 * limit_cycles must lie in [1, 2^31); QNN_EINVAL otherwise.  Read the result
 * with qnn_device_status(stream).
 */
qnn_status qnn_selftest_wait_timeout(int64_t limit_cycles, void *stream);

/* Static description of a status code. */
const char *qnn_status_string(qnn_status s);

/* Library version, for ABI checks: major * 10000 + minor * 100 + patch. */
int32_t qnn_version(void);

#ifdef __cplusplus
}
#endif

#endif /* QNN_H */
