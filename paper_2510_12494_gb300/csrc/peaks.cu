// Roofline denominators that the fp32 kernels are measured against: the FP32
// FMA (SIMT) peak and the TF32 warp-MMA peak of this device, from two
// throughput kernels.  (The bf16 tensor peak and the HBM bandwidth come from
// a cuBLAS GEMM and a copy, measured outside this library.)
#include <cuda_runtime.h>

#include "vfl.h"
#include "vfl_kernels.cuh"

namespace vfl {
namespace {

constexpr int kPeakThreads = 256;

// Eight independent FMA chains per thread; the result is stored so that nothing is dead.
__global__ void __launch_bounds__(kPeakThreads) ffma_kernel(long long iters, float* out) {
    float a[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) a[j] = threadIdx.x * 1e-3f + j;
    const float x = 0.999f, y = 1e-4f;
    for (long long i = 0; i < iters; ++i) {
#pragma unroll
        for (int j = 0; j < 8; ++j) a[j] = fmaf(a[j], x, y);
    }
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) s += a[j];
    out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

__device__ __forceinline__ uint32_t to_tf32(float x) {
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return r;
}

// Eight independent m16n8k8 TF32 MMA accumulators per warp.
__global__ void __launch_bounds__(kPeakThreads) tf32_mma_kernel(long long iters, float* out) {
    uint32_t a[4], b[2];
#pragma unroll
    for (int j = 0; j < 4; ++j) a[j] = to_tf32(1.0f + threadIdx.x * 1e-3f + j);
    b[0] = to_tf32(1e-3f);
    b[1] = to_tf32(2e-3f);
    float d[8][4];
#pragma unroll
    for (int c = 0; c < 8; ++c)
#pragma unroll
        for (int j = 0; j < 4; ++j) d[c][j] = 0.f;
    for (long long i = 0; i < iters; ++i) {
#pragma unroll
        for (int c = 0; c < 8; ++c)
            asm volatile(
                "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                "{%0,%1,%2,%3};"
                : "+f"(d[c][0]), "+f"(d[c][1]), "+f"(d[c][2]), "+f"(d[c][3])
                : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
    }
    float s = 0.f;
#pragma unroll
    for (int c = 0; c < 8; ++c) s += d[c][0] + d[c][1] + d[c][2] + d[c][3];
    out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

}  // namespace
}  // namespace vfl

using namespace vfl;

extern "C" vfl_status vfl_measure_peak(int32_t kind, int64_t iters, double* flops, float* ms) {
    if (!flops || !ms || iters < 1 || (kind != VFL_PEAK_FFMA && kind != VFL_PEAK_TF32_MMA)) {
        set_global_error("vfl_measure_peak: unknown kind, null output or iters < 1");
        return VFL_E_INVAL;
    }
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        set_global_error("vfl_measure_peak: no device");
        return VFL_E_CUDA;
    }
    const int blocks = sms * 8;   // eight resident blocks of 256 threads per SM
    const long long threads = (long long)blocks * kPeakThreads;
    float* out = nullptr;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    cudaError_t e = cudaMalloc(&out, threads * sizeof(float));
    if (e == cudaSuccess) e = cudaEventCreate(&e0);
    if (e == cudaSuccess) e = cudaEventCreate(&e1);
    if (e == cudaSuccess) {
        // one warm-up launch, then the timed one
        for (int rep = 0; rep < 2 && e == cudaSuccess; ++rep) {
            if (rep == 1) cudaEventRecord(e0, 0);
            if (kind == VFL_PEAK_FFMA)
                ffma_kernel<<<blocks, kPeakThreads>>>(iters, out);
            else
                tf32_mma_kernel<<<blocks, kPeakThreads>>>(iters, out);
            e = cudaGetLastError();
        }
        if (e == cudaSuccess) e = cudaEventRecord(e1, 0);
        if (e == cudaSuccess) e = cudaEventSynchronize(e1);
        if (e == cudaSuccess) e = cudaEventElapsedTime(ms, e0, e1);
    }
    if (kind == VFL_PEAK_FFMA)
        *flops = 2.0 * 8.0 * (double)iters * (double)threads;                  // 8 FMAs a thread per iteration
    else
        *flops = 2.0 * 16 * 8 * 8 * 8.0 * (double)iters * (double)(threads / 32);   // 8 m16n8k8 MMAs a warp
    if (e0) cudaEventDestroy(e0);
    if (e1) cudaEventDestroy(e1);
    if (out) cudaFree(out);
    if (e != cudaSuccess) {
        set_global_error(cudaGetErrorString(e));
        return VFL_E_CUDA;
    }
    return VFL_OK;
}
