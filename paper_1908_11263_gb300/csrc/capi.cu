// C ABI of libqnn (declared in include/qnn.h): argument validation, kernel
// selection and the device status word.  Every check happens before anything
// is enqueued; a call that returns an error has launched nothing.
#include <cstdint>
#include <mutex>
#include <vector>

#include "device.cuh"
#include "internal.h"
#include "qnn.h"

namespace qnn {

__device__ int g_status = 0;

int *device_status_ptr()
{
    static std::mutex mu;
    static std::vector<int *> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (dev >= static_cast<int>(cache.size())) cache.resize(dev + 1, nullptr);
    if (!cache[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status) != cudaSuccess) return nullptr;
        cache[dev] = static_cast<int *>(p);
    }
    return cache[dev];
}

int device_sm_count()
{
    static std::mutex mu;
    static std::vector<int> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    std::lock_guard<std::mutex> lock(mu);
    if (dev >= static_cast<int>(cache.size())) cache.resize(dev + 1, 0);
    if (cache[dev] == 0) {
        int sms = 0;
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) sms = 1;
        cache[dev] = sms;
    }
    return cache[dev];
}

namespace {

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }
bool bits_ok(int bits) { return bits == 8 || bits == 4 || bits == 2; }

// Largest im2col length whose worst-case accumulator stays below 2^30, leaving
// 2^30 of headroom for the bias: K * (2^Q - 1) * 2^(Q-1) < 2^30.
bool acc_bound_ok(long long k, int bits)
{
    const long long per = static_cast<long long>((1 << bits) - 1) * (1 << (bits - 1));
    return k * per < (1ll << 30);
}

qnn_status check_conv(const qnn_conv_desc *d, ConvShape *s)
{
    if (!d || d->struct_size != sizeof(qnn_conv_desc)) return QNN_EINVAL;
    if (d->n < 0 || d->h <= 0 || d->w <= 0 || d->c <= 0 || d->m <= 0 || d->kh <= 0 || d->kw <= 0) return QNN_EINVAL;
    if (d->stride_h <= 0 || d->stride_w <= 0 || d->pad_h < 0 || d->pad_w < 0) return QNN_EINVAL;
    if (d->h + 2 * d->pad_h < d->kh || d->w + 2 * d->pad_w < d->kw) return QNN_EINVAL;
    if (d->algo < QNN_ALGO_AUTO || d->algo > QNN_ALGO_TC_GENERAL) return QNN_EINVAL;
    if (!bits_ok(d->bits)) return QNN_EUNSUPPORTED;
    const int per = 8 / d->bits;
    if (d->c % per || d->m % per) return QNN_EUNSUPPORTED;
    if (!acc_bound_ok(static_cast<long long>(d->kh) * d->kw * d->c, d->bits)) return QNN_EUNSUPPORTED;
    s->n = d->n; s->h = d->h; s->w = d->w; s->c = d->c; s->m = d->m; s->kh = d->kh; s->kw = d->kw;
    s->sh = d->stride_h; s->sw = d->stride_w; s->ph = d->pad_h; s->pw = d->pad_w; s->bits = d->bits;
    s->thr = 0;
    s->pool = 0;
    s->oh = (d->h + 2 * d->pad_h - d->kh) / d->stride_h + 1;
    s->ow = (d->w + 2 * d->pad_w - d->kw) / d->stride_w + 1;
    return QNN_OK;
}

// Which kernel serves a descriptor.  Tensor-core requests (QNN_ALGO_AUTO,
// QNN_ALGO_TENSORCORE) take the window kernel when its plan fits the shape,
// else the general tensor-core kernel; QNN_ALGO_TC_WINDOW and
// QNN_ALGO_TC_GENERAL force one of them.
enum Kernel { kDirect = 1, kWindow = 3, kGeneral = 4 };

struct Choice {
    int kernel;  // Kernel, or a negative qnn_status
    TcPlan plan;
    WinPlan wplan;
};

Choice choose(const qnn_conv_desc *d, const ConvShape &s)
{
    Choice c;
    c.plan = plan_conv_tc(s);
    c.wplan = plan_conv_win(s);
    switch (d->algo) {
        case QNN_ALGO_DIRECT: c.kernel = kDirect; break;
        case QNN_ALGO_TC_WINDOW: c.kernel = c.wplan.ok ? kWindow : -QNN_EUNSUPPORTED; break;
        case QNN_ALGO_TC_GENERAL: c.kernel = c.plan.ok ? kGeneral : -QNN_EUNSUPPORTED; break;
        case QNN_ALGO_TENSORCORE:
            c.kernel = c.wplan.ok ? kWindow : c.plan.ok ? kGeneral : -QNN_EUNSUPPORTED;
            break;
        default: c.kernel = c.wplan.ok ? kWindow : c.plan.ok ? kGeneral : kDirect; break;
    }
    return c;
}

// QNN_ALGO_DIRECT or QNN_ALGO_TENSORCORE (either tensor-core kernel), or a negative status.
int choose_algo(const qnn_conv_desc *d, const ConvShape &s, TcPlan *plan)
{
    const Choice c = choose(d, s);
    *plan = c.plan;
    if (c.kernel < 0) return c.kernel;
    return c.kernel == kDirect ? QNN_ALGO_DIRECT : QNN_ALGO_TENSORCORE;
}

qnn_status from_cuda(cudaError_t e) { return e == cudaSuccess ? QNN_OK : QNN_ECUDA; }

// Filters and compression constants; also resolves the algorithm (negative = error).
qnn_status check_params(const qnn_conv_desc *d, const ConvShape &s, const void *w, const int32_t *bias,
                        const int16_t *kappa, const int32_t *lambda, const uint8_t *shifts, TcPlan *plan)
{
    if (!w || !kappa || !lambda) return QNN_EINVAL;
    if (!shifts && (d->shift < 0 || d->shift > 62)) return QNN_EINVAL;
    if (!aligned(w, 16) || !aligned(bias, 4) || !aligned(kappa, 2) || !aligned(lambda, 4)) return QNN_EALIGN;
    const int algo = choose_algo(d, s, plan);
    if (algo < 0) return static_cast<qnn_status>(-algo);
    return QNN_OK;
}

qnn_status check_workspace(const TcPlan &plan, const void *workspace, size_t bytes)
{
    if (!workspace || bytes < plan.workspace_bytes || !aligned(workspace, 256)) return QNN_EWORKSPACE;
    return QNN_OK;
}

// Scratch of qconv_hwc_noalloc(): part of the library's device image, so that
// entry point never allocates.  Each device that loads the library holds its own
// copy until exit.  In host code the name is only a stand-in for the symbol;
// the device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_noalloc_scratch[QNN_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

// Device address of g_noalloc_scratch on the current device, looked up on the
// first call per device (with that device current); nullptr on failure.  The
// cache is a fixed array, so this allocates no memory on host or device.
void *noalloc_scratch_ptr()
{
    static std::mutex mu;
    static void *cache[kMaxDevices] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!cache[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
        cache[dev] = p;
    }
    return cache[dev];
}

// One warp waits on a barrier that nothing arrives on (bounded by `limit`).
__global__ void selftest_timeout_kernel(int *status, long long limit)
{
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_mbar_init();
    }
    __syncwarp();
    mbar_wait_warp(&bar, 0, status, limit);
}

}  // namespace
}  // namespace qnn

using namespace qnn;

extern "C" {

qnn_status qconv_hwc_workspace_size(const qnn_conv_desc *d, size_t *bytes)
{
    if (!bytes) return QNN_EINVAL;
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return st;
    const Choice c = choose(d, s);
    if (c.kernel < 0) return static_cast<qnn_status>(-c.kernel);
    *bytes = c.kernel == kWindow ? c.wplan.img_bytes : c.kernel == kGeneral ? c.plan.workspace_bytes : 0;
    return QNN_OK;
}

int32_t qconv_hwc_tc_kernel(const qnn_conv_desc *d)
{
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return -static_cast<int32_t>(st);
    const Choice c = choose(d, s);
    if (c.kernel < 0) return c.kernel;
    return c.kernel == kDirect ? 0 : c.kernel;
}

int32_t qconv_hwc_algo(const qnn_conv_desc *d)
{
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return -static_cast<int32_t>(st);
    TcPlan plan;
    return choose_algo(d, s, &plan);
}

int32_t qconv_hwc_mma_operand_bits(const qnn_conv_desc *d)
{
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return -static_cast<int32_t>(st);
    const Choice c = choose(d, s);
    if (c.kernel < 0) return c.kernel;
    if (c.kernel == kWindow) return c.wplan.fp8 ? 8 : 16;
    if (c.kernel == kGeneral) return c.plan.fp8 ? 8 : 16;
    return 0;
}

qnn_status qconv_hwc_prepare(const qnn_conv_desc *d, const void *w, const int32_t *bias, const int16_t *kappa,
                             const int32_t *lambda, const uint8_t *shifts, void *workspace, size_t workspace_bytes,
                             void *stream)
{
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return st;
    TcPlan plan;
    st = check_params(d, s, w, bias, kappa, lambda, shifts, &plan);
    if (st != QNN_OK) return st;
    const Choice c = choose(d, s);
    if (c.kernel == kDirect) return QNN_OK;
    ConvParams p{nullptr, static_cast<const uint8_t *>(w), bias, kappa, lambda, shifts, d->shift, nullptr};
    if (c.kernel == kWindow) {
        if (!workspace || workspace_bytes < c.wplan.img_bytes || !aligned(workspace, 256)) return QNN_EWORKSPACE;
        return from_cuda(prepare_conv_win(c.wplan, s, p, workspace, static_cast<cudaStream_t>(stream)));
    }
    st = check_workspace(plan, workspace, workspace_bytes);
    if (st != QNN_OK) return st;
    return from_cuda(launch_conv_tc_prep(plan, s, p, workspace, static_cast<cudaStream_t>(stream)));
}

qnn_status qconv_hwc_run(const qnn_conv_desc *d, const void *x, void *y, const void *workspace,
                         size_t workspace_bytes, void *stream)
{
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return st;
    if (s.n > 0 && (!x || !y)) return QNN_EINVAL;
    if (!aligned(x, 16) || !aligned(y, 16)) return QNN_EALIGN;
    const Choice c = choose(d, s);
    if (c.kernel < 0) return static_cast<qnn_status>(-c.kernel);
    if (c.kernel == kDirect) return QNN_EUNSUPPORTED;
    if (c.kernel == kWindow) {
        if (!workspace || workspace_bytes < c.wplan.img_bytes || !aligned(workspace, 256)) return QNN_EWORKSPACE;
        ConvParams p{};
        p.x = static_cast<const uint8_t *>(x);
        p.y = static_cast<uint8_t *>(y);
        return from_cuda(launch_conv_win(c.wplan, s, p, static_cast<cudaStream_t>(stream), workspace));
    }
    st = check_workspace(c.plan, workspace, workspace_bytes);
    if (st != QNN_OK) return st;
    return from_cuda(launch_conv_tc_run(c.plan, s, static_cast<const uint8_t *>(x), static_cast<uint8_t *>(y),
                                        workspace, static_cast<cudaStream_t>(stream), false));
}

qnn_status qconv_hwc(const qnn_conv_desc *d, const void *x, const void *w, const int32_t *bias, const int16_t *kappa,
                     const int32_t *lambda, const uint8_t *shifts, void *y, void *workspace, size_t workspace_bytes,
                     void *stream)
{
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return st;
    if (s.n > 0 && (!x || !y)) return QNN_EINVAL;
    if (!aligned(x, 16) || !aligned(y, 16)) return QNN_EALIGN;
    TcPlan plan;
    st = check_params(d, s, w, bias, kappa, lambda, shifts, &plan);
    if (st != QNN_OK) return st;
    const Choice c = choose(d, s);
    cudaStream_t cs = static_cast<cudaStream_t>(stream);
    if (c.kernel == kWindow) {  // one launch; the filters are read where the caller keeps them
        ConvParams p{static_cast<const uint8_t *>(x), static_cast<const uint8_t *>(w), bias, kappa, lambda, shifts,
                     d->shift, static_cast<uint8_t *>(y)};
        return from_cuda(launch_conv_win(c.wplan, s, p, cs));
    }
    if (c.kernel == kGeneral) {
        st = check_workspace(plan, workspace, workspace_bytes);
        if (st != QNN_OK) return st;
        ConvParams p{static_cast<const uint8_t *>(x), static_cast<const uint8_t *>(w), bias, kappa, lambda, shifts,
                     d->shift, static_cast<uint8_t *>(y)};
        cudaError_t e = launch_conv_tc_prep(plan, s, p, workspace, cs);
        if (e == cudaSuccess) e = launch_conv_tc_run(plan, s, p.x, p.y, workspace, cs, true);
        return from_cuda(e);
    }
    if (s.n == 0) return QNN_OK;
    ConvParams p{static_cast<const uint8_t *>(x), static_cast<const uint8_t *>(w), bias, kappa, lambda, shifts,
                 d->shift, static_cast<uint8_t *>(y)};
    return from_cuda(launch_conv_direct(s, p, cs));
}

qnn_status qconv_hwc_pool2(const qnn_conv_desc *d, const void *x, const void *w, const int32_t *bias,
                           const int16_t *kappa, const int32_t *lambda, const uint8_t *shifts, void *y, void *workspace,
                           size_t workspace_bytes, void *stream)
{
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return st;
    if (s.oh < 2 || s.ow < 2) return QNN_EINVAL;  // no pooled pixel
    s.pool = 1;
    if (s.n > 0 && (!x || !y)) return QNN_EINVAL;
    if (!aligned(x, 16) || !aligned(y, 16)) return QNN_EALIGN;
    TcPlan plan;
    st = check_params(d, s, w, bias, kappa, lambda, shifts, &plan);
    if (st != QNN_OK) return st;
    // the fused pool runs in the tensor-core kernels only (strip tiles)
    const Choice c = choose(d, s);
    cudaStream_t cs = static_cast<cudaStream_t>(stream);
    ConvParams p{static_cast<const uint8_t *>(x), static_cast<const uint8_t *>(w), bias, kappa, lambda, shifts,
                 d->shift, static_cast<uint8_t *>(y)};
    if (c.kernel == kWindow) return from_cuda(launch_conv_win(c.wplan, s, p, cs));
    if (c.kernel != kGeneral || !plan.strip) return QNN_EUNSUPPORTED;
    st = check_workspace(plan, workspace, workspace_bytes);
    if (st != QNN_OK) return st;
    cudaError_t e = launch_conv_tc_prep(plan, s, p, workspace, cs);
    if (e == cudaSuccess) e = launch_conv_tc_run(plan, s, p.x, p.y, workspace, cs, true);
    return from_cuda(e);
}

qnn_status qconv_hwc_pool2_run(const qnn_conv_desc *d, const void *x, void *y, const void *workspace,
                               size_t workspace_bytes, void *stream)
{
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return st;
    if (s.oh < 2 || s.ow < 2) return QNN_EINVAL;  // no pooled pixel
    if (s.n > 0 && (!x || !y)) return QNN_EINVAL;
    if (!aligned(x, 16) || !aligned(y, 16)) return QNN_EALIGN;
    // the kernel and plan qconv_hwc_prepare chose for this descriptor (the window
    // planner's layout does not depend on the fused pool)
    const Choice c = choose(d, s);
    if (c.kernel < 0) return static_cast<qnn_status>(-c.kernel);
    if (c.kernel != kWindow) return QNN_EUNSUPPORTED;
    if (!workspace || workspace_bytes < c.wplan.img_bytes || !aligned(workspace, 256)) return QNN_EWORKSPACE;
    s.pool = 1;
    ConvParams p{};
    p.x = static_cast<const uint8_t *>(x);
    p.y = static_cast<uint8_t *>(y);
    return from_cuda(launch_conv_win(c.wplan, s, p, static_cast<cudaStream_t>(stream), workspace));
}

qnn_status qconv_hwc_thresholds(const qnn_conv_desc *d, const void *x, const void *w, const int32_t *thresholds,
                                void *y, void *workspace, size_t workspace_bytes, void *stream)
{
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return st;
    if (s.bits == 8) return QNN_EUNSUPPORTED;  // INT-8 outputs use scaling and clipping (qconv_hwc)
    s.thr = 1;
    if (s.n > 0 && (!x || !y)) return QNN_EINVAL;
    if (!w || !thresholds) return QNN_EINVAL;
    if (!aligned(x, 16) || !aligned(y, 16) || !aligned(w, 16) || !aligned(thresholds, 4)) return QNN_EALIGN;
    TcPlan plan;
    const int algo = choose_algo(d, s, &plan);
    if (algo < 0) return static_cast<qnn_status>(-algo);
    const Choice c = choose(d, s);
    cudaStream_t cs = static_cast<cudaStream_t>(stream);
    ConvParams p{static_cast<const uint8_t *>(x), static_cast<const uint8_t *>(w), nullptr, nullptr, nullptr, nullptr,
                 0, static_cast<uint8_t *>(y), thresholds};
    if (c.kernel == kWindow) return from_cuda(launch_conv_win(c.wplan, s, p, cs));
    if (algo == QNN_ALGO_TENSORCORE) {
        st = check_workspace(plan, workspace, workspace_bytes);
        if (st != QNN_OK) return st;
        cudaError_t e = launch_conv_tc_prep(plan, s, p, workspace, cs);
        if (e == cudaSuccess) e = launch_conv_tc_run(plan, s, p.x, p.y, workspace, cs, true);
        return from_cuda(e);
    }
    if (s.n == 0) return QNN_OK;
    return from_cuda(launch_conv_direct(s, p, cs));
}

qnn_status qconv_hwc_binary(const qnn_conv_desc *d, const void *x, const void *w, const int32_t *thresholds, void *y,
                            void *stream)
{
    if (!d || d->struct_size != sizeof(qnn_conv_desc)) return QNN_EINVAL;
    if (d->n < 0 || d->h <= 0 || d->w <= 0 || d->c <= 0 || d->m <= 0 || d->kh <= 0 || d->kw <= 0) return QNN_EINVAL;
    if (d->stride_h <= 0 || d->stride_w <= 0 || d->pad_h < 0 || d->pad_w < 0) return QNN_EINVAL;
    if (d->h + 2 * d->pad_h < d->kh || d->w + 2 * d->pad_w < d->kw) return QNN_EINVAL;
    if (d->bits != 1 || d->c % 8 || d->m % 8) return QNN_EUNSUPPORTED;
    if (static_cast<long long>(d->kh) * d->kw * d->c >= (1ll << 31)) return QNN_EUNSUPPORTED;
    if (!w || !thresholds || (d->n > 0 && (!x || !y))) return QNN_EINVAL;
    if (!aligned(thresholds, 4)) return QNN_EALIGN;
    ConvShape s{};
    s.n = d->n; s.h = d->h; s.w = d->w; s.c = d->c; s.m = d->m; s.kh = d->kh; s.kw = d->kw;
    s.sh = d->stride_h; s.sw = d->stride_w; s.ph = d->pad_h; s.pw = d->pad_w; s.bits = 1;
    s.oh = (d->h + 2 * d->pad_h - d->kh) / d->stride_h + 1;
    s.ow = (d->w + 2 * d->pad_w - d->kw) / d->stride_w + 1;
    return from_cuda(launch_conv_binary(s, static_cast<const uint8_t *>(x), static_cast<const uint8_t *>(w), thresholds,
                                        static_cast<uint8_t *>(y), static_cast<cudaStream_t>(stream)));
}

qnn_status qconv_hwc_noalloc(const qnn_conv_desc *d, const void *x, const void *w, const int32_t *bias,
                             const int16_t *kappa, const int32_t *lambda, const uint8_t *shifts, void *y,
                             void *stream)
{
    ConvShape s;
    qnn_status st = check_conv(d, &s);
    if (st != QNN_OK) return st;
    if (s.n > 0 && (!x || !y)) return QNN_EINVAL;
    if (!aligned(x, 16) || !aligned(y, 16)) return QNN_EALIGN;
    TcPlan plan;
    st = check_params(d, s, w, bias, kappa, lambda, shifts, &plan);
    if (st != QNN_OK) return st;
    // this entry point runs the general tensor-core kernel, whose prepared filters go to the scratch array
    if (choose_algo(d, s, &plan) != QNN_ALGO_TENSORCORE || !plan.ok || d->algo == QNN_ALGO_TC_WINDOW)
        return QNN_EUNSUPPORTED;
    if (plan.workspace_bytes > static_cast<size_t>(QNN_NOALLOC_SCRATCH_BYTES)) return QNN_ESCRATCH;
    // an empty batch computes nothing, so it enqueues nothing and leaves the
    // shared scratch array to the calls that use it
    if (s.n == 0) return QNN_OK;
    void *scratch = noalloc_scratch_ptr();
    if (!scratch) return QNN_ECUDA;
    // the prep kernel rewrites every scratch byte the convolution reads, so the
    // previous call's contents never reach this one
    cudaStream_t cs = static_cast<cudaStream_t>(stream);
    ConvParams p{static_cast<const uint8_t *>(x), static_cast<const uint8_t *>(w), bias, kappa, lambda, shifts,
                 d->shift, static_cast<uint8_t *>(y)};
    cudaError_t e = launch_conv_tc_prep(plan, s, p, scratch, cs);
    if (e == cudaSuccess) e = launch_conv_tc_run(plan, s, p.x, p.y, scratch, cs, true);
    return from_cuda(e);
}

qnn_status qlinear(int32_t n, int32_t k, int32_t m, const uint8_t *x, const int8_t *w, const int32_t *bias,
                   int32_t *y, void *stream)
{
    if (n < 0 || k <= 0 || m <= 0) return QNN_EINVAL;
    if (!w || (n > 0 && (!x || !y))) return QNN_EINVAL;
    if (static_cast<long long>(k) * 255 * 128 >= (1ll << 30)) return QNN_EUNSUPPORTED;
    if (!aligned(y, 4) || !aligned(bias, 4)) return QNN_EALIGN;
    return from_cuda(launch_linear(n, k, m, x, w, bias, y, static_cast<cudaStream_t>(stream)));
}

qnn_status qmaxpool(int32_t n, int32_t h, int32_t w, int32_t c, int32_t k, int32_t s, int32_t bits, const void *x,
                    void *y, void *stream)
{
    if (n < 0 || h <= 0 || w <= 0 || c <= 0 || k <= 0 || s <= 0 || k > h || k > w) return QNN_EINVAL;
    if (n > 0 && (!x || !y)) return QNN_EINVAL;
    if (!bits_ok(bits)) return QNN_EUNSUPPORTED;
    if (c % (8 / bits)) return QNN_EUNSUPPORTED;
    return from_cuda(launch_maxpool(n, h, w, c, k, s, bits, static_cast<const uint8_t *>(x),
                                    static_cast<uint8_t *>(y), static_cast<cudaStream_t>(stream)));
}

qnn_status pack_subbyte(const int8_t *src, void *dst, int64_t count, int32_t bits, void *stream)
{
    if (count < 0) return QNN_EINVAL;
    if (count > 0 && (!src || !dst)) return QNN_EINVAL;
    if (!bits_ok(bits)) return QNN_EUNSUPPORTED;
    if (count % (8 / bits)) return QNN_EUNSUPPORTED;
    return from_cuda(launch_pack(src, static_cast<uint8_t *>(dst), count, bits, static_cast<cudaStream_t>(stream)));
}

qnn_status unpack_subbyte(const void *src, int8_t *dst, int64_t count, int32_t bits, int32_t is_signed, void *stream)
{
    if (count < 0) return QNN_EINVAL;
    if (count > 0 && (!src || !dst)) return QNN_EINVAL;
    if (!bits_ok(bits)) return QNN_EUNSUPPORTED;
    if (count % (8 / bits)) return QNN_EUNSUPPORTED;
    return from_cuda(launch_unpack(static_cast<const uint8_t *>(src), dst, count, bits, is_signed ? 1 : 0,
                                   static_cast<cudaStream_t>(stream)));
}

qnn_status qnn_selftest_wait_timeout(int64_t limit_cycles, void *stream)
{
    if (limit_cycles < 1 || limit_cycles >= (1ll << 31)) return QNN_EINVAL;
    int *status = device_status_ptr();
    if (!status) return QNN_ECUDA;
    selftest_timeout_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(status, limit_cycles);
    return from_cuda(cudaGetLastError());
}

qnn_status qnn_device_status(void *stream)
{
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return QNN_ECUDA;
    int v = 0;
    if (cudaMemcpyFromSymbol(&v, g_status, sizeof(int)) != cudaSuccess) return QNN_ECUDA;
    const int zero = 0;
    if (v != 0 && cudaMemcpyToSymbol(g_status, &zero, sizeof(int)) != cudaSuccess) return QNN_ECUDA;
    return static_cast<qnn_status>(v);
}

const char *qnn_status_string(qnn_status s)
{
    switch (s) {
        case QNN_OK: return "ok";
        case QNN_EINVAL: return "invalid argument";
        case QNN_EUNSUPPORTED: return "unsupported configuration";
        case QNN_EALIGN: return "misaligned pointer";
        case QNN_ECUDA: return "CUDA error";
        case QNN_ETIMEOUT: return "device-side wait timed out";
        case QNN_EWORKSPACE: return "workspace missing or too small";
        case QNN_ESCRATCH: return "layer needs more scratch than the no-allocation entry point's fixed array holds";
        default: return "unknown status";
    }
}

int32_t qnn_version(void) { return 100; }

}  // extern "C"
