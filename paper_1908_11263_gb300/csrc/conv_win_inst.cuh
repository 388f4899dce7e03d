// Instantiations of the window kernel for one bit width (QNN_WIN_BITS), by
// output-channel tile, fused pool and (INT-8, at most 64 filters) folded
// kernel columns.  Included once by each conv_win_q*.cu.
#pragma once

#include <mutex>

#include "conv_win.cuh"

#ifndef QNN_WIN_BITS
#error "define QNN_WIN_BITS (8, 4 or 2) before including conv_win_inst.cuh"
#endif

namespace qnn {
namespace {

template <int BITS, int NT, bool POOL, bool FOLD = false>
cudaError_t launch_one(const win::WinArgs &a, int grid, uint32_t smem, cudaStream_t st)
{
    // the opt-in shared-memory limit is raised once per device, outside any stream capture
    static std::mutex mu;
    static bool raised[64] = {};
    auto kern = win::conv_win_kernel<BITS, NT, POOL, FOLD>;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
        if (!raised[dev]) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, win::kSmemLimit);
            if (e != cudaSuccess) return e;
            raised[dev] = true;
        }
    }
    // launched with programmatic stream serialization: the kernel lets its
    // successor launch early and waits for its predecessor before reading memory
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(win::kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

}  // namespace

template <>
cudaError_t launch_win_bits<QNN_WIN_BITS>(const win::WinArgs &a, int nt, int grid, uint32_t smem, cudaStream_t st)
{
    constexpr int B = QNN_WIN_BITS;
#if QNN_WIN_BITS == 8
    // folded plans (few input channels) have their own instantiations, at most 64 filters
    if (a.fold) {
        switch (nt) {
            case 32: return a.pool ? launch_one<B, 32, true, true>(a, grid, smem, st)
                                   : launch_one<B, 32, false, true>(a, grid, smem, st);
            case 64: return a.pool ? launch_one<B, 64, true, true>(a, grid, smem, st)
                                   : launch_one<B, 64, false, true>(a, grid, smem, st);
            default: return cudaErrorInvalidValue;
        }
    }
#endif
    switch (nt) {
        case 32: return a.pool ? launch_one<B, 32, true>(a, grid, smem, st) : launch_one<B, 32, false>(a, grid, smem, st);
        case 64: return a.pool ? launch_one<B, 64, true>(a, grid, smem, st) : launch_one<B, 64, false>(a, grid, smem, st);
        case 128:
            return a.pool ? launch_one<B, 128, true>(a, grid, smem, st) : launch_one<B, 128, false>(a, grid, smem, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace qnn
