// Allocation-free weight gradient of one Linear layer.
//
// Some callers cannot allocate device memory at the point where they need
// this: code running inside an allocator or memory-pool callback, code that
// has promised its host a fixed device footprint, or a process that has
// already reserved every byte of HBM for its own pools.  For them the library
// keeps one fixed scratch area in a file-scope __device__ array, so this entry
// point needs no workspace from the caller and calls no allocating routine.
#include <algorithm>
#include <cstring>
#include <mutex>
#include <string>

#include "vfl_kernels.cuh"

namespace vfl {

namespace {

// Split-K partial sums of dW and db.  Every GPU that loads the library holds
// this array until the process exits.
constexpr unsigned long long kNoAllocScratchBytes = 16ull << 20;   // 16 MiB
constexpr long long kNoAllocScratchFloats = (long long)(kNoAllocScratchBytes / sizeof(float));
static __device__ __align__(256) float g_noalloc_scratch[kNoAllocScratchFloats];

// Device address of g_noalloc_scratch and the device's SM count, looked up
// once per device.  In host code the array's name is only a host-side
// stand-in, so kernels must be given this address instead.  The address is
// cached for the life of the process: a device reset (cudaDeviceReset) after
// the first call is not supported.
constexpr int kMaxDevices = 64;
std::mutex g_mu;
float* g_scratch_ptr[kMaxDevices] = {};
int g_sm_count[kMaxDevices] = {};

// The SIMT GEMM tiles the layer's inputs in blocks of 64 along grid.y.
constexpr long long kMaxIn = 65535LL * 64;

// dW[i] = sum_z P[z * stride + i] (i < n_w); db[j] = sum_z Pb[z * n_b + j], in z order.
__global__ void reduce_partials_kernel(const float* __restrict__ P, long long stride, long long n_w,
                                       const float* __restrict__ Pb, int n_b, int nsplit, float* __restrict__ dW,
                                       float* __restrict__ db) {
    const long long n = n_w + n_b;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        float a = 0.f;
        if (i < n_w) {
            for (int z = 0; z < nsplit; ++z) a += P[z * stride + i];
            dW[i] = a;
        } else {
            const long long j = i - n_w;
            for (int z = 0; z < nsplit; ++z) a += Pb[(long long)z * n_b + j];
            db[j] = a;
        }
    }
}

}  // namespace

}  // namespace vfl

using namespace vfl;

extern "C" vfl_status vfl_weight_grad_noalloc(const void* dpre, const void* x, int32_t rows, int32_t out, int32_t in,
                                              int32_t dtype, float* dW, float* db, void* stream) {
    if (!dpre || !x || !dW || !db || rows < 1 || out < 1 || in < 1 || (dtype != VFL_FP32 && dtype != VFL_BF16)) {
        set_global_error("vfl_weight_grad_noalloc: null pointer, non-positive size or unknown dtype");
        return VFL_E_INVAL;
    }
    // Split the row reduction so that the partials fit the fixed scratch area.
    const long long per_split = (long long)out * in + out;
    if (per_split > kNoAllocScratchFloats) {
        set_global_error(("vfl_weight_grad_noalloc: a " + std::to_string(out) + "x" + std::to_string(in) +
                          " layer needs more than the fixed scratch of " + std::to_string(kNoAllocScratchBytes >> 20) +
                          " MiB (out*in + out must be at most " + std::to_string(kNoAllocScratchFloats) + ")")
                             .c_str());
        return VFL_E_INVAL;
    }
    if (in > kMaxIn) {
        set_global_error(("vfl_weight_grad_noalloc: in = " + std::to_string(in) + " exceeds the largest supported "
                          "input width " + std::to_string(kMaxIn)).c_str());
        return VFL_E_INVAL;
    }

    // One-time set-up on the current device: the scratch array's device address and the SM count.
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
        set_global_error((std::string("vfl_weight_grad_noalloc: no usable current device: ") + cudaGetErrorString(e)).c_str());
        return VFL_E_CUDA;
    }
    float* scratch = nullptr;
    int sm_count = 0;
    {
        std::lock_guard<std::mutex> lock(g_mu);
        if (!g_scratch_ptr[dev]) {
            void* p = nullptr;
            e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
            if (e != cudaSuccess || !p) {
                set_global_error((std::string("vfl_weight_grad_noalloc: cudaGetSymbolAddress failed: ") +
                                  cudaGetErrorString(e)).c_str());
                return VFL_E_CUDA;
            }
            int sms = 0;
            e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            if (e != cudaSuccess || sms < 1) {
                set_global_error((std::string("vfl_weight_grad_noalloc: SM count query failed: ") +
                                  cudaGetErrorString(e)).c_str());
                return VFL_E_CUDA;
            }
            g_sm_count[dev] = sms;
            g_scratch_ptr[dev] = static_cast<float*>(p);
        }
        scratch = g_scratch_ptr[dev];
        sm_count = g_sm_count[dev];
    }
    // Split the rows so that about two blocks per SM run, within the scratch.
    const long long tiles = (long long)((out + 63) / 64) * ((in + 63) / 64);
    long long nsplit = std::max<long long>(1, 2LL * sm_count / std::max<long long>(1, tiles));
    nsplit = std::min<long long>(nsplit, std::max(1, rows / 64));
    nsplit = std::min<long long>(nsplit, 32);
    nsplit = std::min<long long>(nsplit, kNoAllocScratchFloats / per_split);
    const int kchunk = (int)(((rows + nsplit - 1) / nsplit + 15) / 16 * 16);
    nsplit = (rows + kchunk - 1) / kchunk;
    float* P = scratch;
    float* Pb = scratch + nsplit * (long long)out * in;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int bf = dtype == VFL_BF16;

    // dW[out, in] = dpre^T x and db = column sums of dpre, split over row chunks;
    // every partial is written (zeros where a chunk is empty), so nothing in the
    // scratch has to start at zero.
    GemmArgs g;
    memset(&g, 0, sizeof g);
    g.mode = GEMM_DW;
    g.M = out;
    g.N = in;
    g.K = rows;
    g.n_split = in;
    g.A = dpre; g.a_rs = 1; g.a_cs = out;
    g.B = x; g.b_rs = 1; g.b_cs = in;
    g.P = P; g.p_stride = (long long)out * in; g.ldc = in;
    g.Pb = Pb; g.pb_stride = out;
    g.kchunk = kchunk;
    e = launch_gemm_simt(g, bf, bf, bf, (int)nsplit, s);
    if (e == cudaSuccess) {
        const long long n = (long long)out * in + out;
        long long blocks = std::min<long long>((n + 255) / 256, (long long)sm_count * 8);
        reduce_partials_kernel<<<(int)blocks, 256, 0, s>>>(P, (long long)out * in, (long long)out * in, Pb, out,
                                                            (int)nsplit, dW, db);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) {
        set_global_error((std::string("vfl_weight_grad_noalloc: launch failed: ") + cudaGetErrorString(e)).c_str());
        return VFL_E_CUDA;
    }
    return VFL_OK;
}

