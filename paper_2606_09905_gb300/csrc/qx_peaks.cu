// qx_peaks.cu -- a measurement utility, not part of any operator: the
// throughput of the legacy warp-level INT8 tensor instruction on this device.
//
// The INT16 GEMM of Table 1 could be built from INT8 limbs (a = 256 a_hi +
// a_lo, four s8 x s8 -> s32 products per INT16 product).  sm_103a has no
// tcgen05 INT8 kind, so the only INT8 tensor path is the warp-level
// mma.sync.m16n8k32 s8 instruction.  Its measured peak divided by four is the
// roofline an INT8-limb design would have, reported beside the FP16-digit
// substrate's own roofline.
//
// Each warp runs long chains of independent MMAs on register-resident
// fragments (no memory traffic in the loop); one value per warp is written at
// the end so the work cannot be removed.
#include <cuda_runtime.h>

#include <cstdint>

#include "qx.h"

namespace {

constexpr int kChains = 8;            // independent accumulators per warp
constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads) int8_mma_peak_kernel(int iters, int32_t *sink) {
    // A: 16 x 32 s8 (4 registers), B: 32 x 8 s8 (2 registers), per thread
    uint32_t a[4], b[2];
    const uint32_t seed = threadIdx.x * 2654435761u + blockIdx.x;
#pragma unroll
    for (int i = 0; i < 4; ++i) a[i] = seed * (2 * i + 1) | 0x01010101u;
#pragma unroll
    for (int i = 0; i < 2; ++i) b[i] = seed * (2 * i + 7) | 0x01010101u;
    int32_t d[kChains][4];
#pragma unroll
    for (int c = 0; c < kChains; ++c)
#pragma unroll
        for (int i = 0; i < 4; ++i) d[c][i] = 0;
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int c = 0; c < kChains; ++c) {
            asm volatile(
                "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 "
                "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};\n"
                : "+r"(d[c][0]), "+r"(d[c][1]), "+r"(d[c][2]), "+r"(d[c][3])
                : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
        }
    }
    int32_t acc = 0;
#pragma unroll
    for (int c = 0; c < kChains; ++c) acc += d[c][0] ^ d[c][1] ^ d[c][2] ^ d[c][3];
    if ((threadIdx.x & 31) == 0) sink[blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5)] = acc;
}

}  // namespace

extern "C" qx_status qx_measure_int8_mma_peak(int device, double *tops) {
    if (!tops) return QX_ERR_INVALID_ARG;
    *tops = 0.0;
    int prev = 0;
    if (cudaGetDevice(&prev) != cudaSuccess || cudaSetDevice(device) != cudaSuccess) {
        cudaGetLastError();
        return QX_ERR_DEVICE;
    }
    cudaDeviceProp prop;
    qx_status st = QX_OK;
    int32_t *sink = nullptr;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    const int iters = 256;
    int blocks = 0;
    float ms = 0.f;
    if (cudaGetDeviceProperties(&prop, device) != cudaSuccess) {
        st = QX_ERR_CUDA;
        goto done;
    }
    blocks = prop.multiProcessorCount * 8;
    if (cudaMalloc(&sink, size_t(blocks) * (kThreads / 32) * sizeof(int32_t)) != cudaSuccess ||
        cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess) {
        st = QX_ERR_CUDA;
        goto done;
    }
    int8_mma_peak_kernel<<<blocks, kThreads>>>(iters / 8, sink);   // warm-up
    cudaEventRecord(e0);
    int8_mma_peak_kernel<<<blocks, kThreads>>>(iters, sink);
    cudaEventRecord(e1);
    if (cudaEventSynchronize(e1) != cudaSuccess || cudaEventElapsedTime(&ms, e0, e1) != cudaSuccess ||
        ms <= 0.f) {
        st = QX_ERR_CUDA;
        goto done;
    }
    {
        // ops per mma.sync m16n8k32: 2 * 16 * 8 * 32
        const double ops = double(blocks) * (kThreads / 32) * iters * kChains * 2.0 * 16 * 8 * 32;
        *tops = ops / (double(ms) * 1e-3) / 1e12;
    }
done:
    cudaGetLastError();
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
    if (sink) cudaFree(sink);
    cudaSetDevice(prev);
    return st;
}
