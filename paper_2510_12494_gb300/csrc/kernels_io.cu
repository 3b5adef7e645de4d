// Host staging of bit-packed binary features.
//
// A party whose features are all 0 / 1 (the wide binary workload: Bernoulli indicator columns) can keep
// them on the host as bits: row r of a [rows, d] matrix is ceil(d / 32) 32-bit words, feature c in bit
// c mod 32 of word c / 32.  Each step's kernel reads its rows' words over the host link (1/16 of the bytes
// of bf16 rows) and writes the slot rows the step's GEMMs read: d values 1.0 or 0.0 (bf16 or fp32) and zeros
// in the padding columns [d, ld).  The values are exact, so a step on bit-packed rows is bit-identical to
// one on the same rows held as bf16 or fp32.
#include <algorithm>

#include "vfl_kernels.cuh"
#include "vfl_pdl.cuh"

namespace vfl {

namespace {

// Blocks of a staging kernel: four per SM pull the host link's full rate and leave the other warp slots to
// the step's compute kernels.
constexpr int kBitsBlocks = 152 * 4;

// 32 features (one host word) as values of T: bf16 1.0 is 0x3F80, fp32 1.0 is 0x3F800000.
template <typename T>
__device__ __forceinline__ void expand_word(uint32_t bits, T* out, int cols);

template <>
__device__ __forceinline__ void expand_word<uint16_t>(uint32_t bits, uint16_t* out, int cols) {
    if (cols == 32) {
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            uint32_t w[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const uint32_t b = bits >> (8 * v + 2 * j);
                w[j] = (b & 1u) * 0x3F80u | ((b >> 1) & 1u) * 0x3F800000u;
            }
            reinterpret_cast<uint4*>(out)[v] = make_uint4(w[0], w[1], w[2], w[3]);
        }
    } else {
        for (int c = 0; c < cols; ++c) out[c] = (bits >> c) & 1u ? 0x3F80u : 0u;
    }
}

template <>
__device__ __forceinline__ void expand_word<uint32_t>(uint32_t bits, uint32_t* out, int cols) {
    if (cols == 32) {
#pragma unroll
        for (int v = 0; v < 8; ++v) {
            const uint32_t b = bits >> (4 * v);
            reinterpret_cast<uint4*>(out)[v] = make_uint4((b & 1u) * 0x3F800000u, ((b >> 1) & 1u) * 0x3F800000u,
                                                          ((b >> 2) & 1u) * 0x3F800000u, ((b >> 3) & 1u) * 0x3F800000u);
        }
    } else {
        for (int c = 0; c < cols; ++c) out[c] = (bits >> c) & 1u ? 0x3F800000u : 0u;
    }
}

// Rows [0, rows) of one party: host words h [rows, ceil(d / 32)] into dst [rows, ld] (ld >= d, a multiple of
// 8, dst 16-byte aligned: every full word's 32 values start on a 64-byte (bf16) or 128-byte (fp32) boundary).
template <typename T>
__device__ __forceinline__ void unpack_rows(const uint32_t* __restrict__ h, int d, int rows, T* dst, long long ld,
                                            int tid, int nthreads) {
    const int wpr = (d + 31) >> 5;
    const long long n = (long long)rows * wpr;
    for (long long i = tid; i < n; i += nthreads) {
        const long long r = i / wpr;
        const int c0 = 32 * (int)(i - r * wpr);
        expand_word<T>(__ldcs(h + i), dst + r * ld + c0, min(32, d - c0));
    }
    const int pad = (int)(ld - d);
    for (long long i = tid; i < (long long)rows * pad; i += nthreads) {
        const long long r = i / pad;
        dst[r * ld + d + (i - r * pad)] = 0;
    }
}

template <typename T>
__global__ void stage_rows_bits_kernel(const uint32_t* __restrict__ hxp, int dp, const uint32_t* __restrict__ hxa,
                                       int da, const int* __restrict__ hy, int rows, T* xp, long long ld_p, T* xa,
                                       long long ld_a, int* __restrict__ y) {
    pdl_entry();
    const int tid = blockIdx.x * blockDim.x + threadIdx.x, nt = gridDim.x * blockDim.x;
    unpack_rows(hxp, dp, rows, xp, ld_p, tid, nt);
    unpack_rows(hxa, da, rows, xa, ld_a, tid, nt);
    for (int i = tid; i < rows; i += nt) y[i] = hy[i];
}

template <typename K>
bool shared_split(K kernel) {
    // the shared-memory-heavy L1 split every kernel of the library asks for (an SM whose split changes
    // between two kernels drains first)
    return cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                (int)cudaSharedmemCarveoutMaxShared) == cudaSuccess;
}

}  // namespace

cudaError_t launch_stage_rows_bits(const uint32_t* hxp, int dp, const uint32_t* hxa, int da, const int* hy, int rows,
                                   void* xp, long long ld_p, void* xa, long long ld_a, int* y, int bf16,
                                   cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    const long long words = (long long)rows * (((dp + 31) >> 5) + ((da + 31) >> 5));
    const int grid = (int)std::max<long long>(1, std::min<long long>((words + 255) / 256, kBitsBlocks));
    if (bf16) {
        static const bool split = shared_split(stage_rows_bits_kernel<uint16_t>);
        (void)split;
        stage_rows_bits_kernel<uint16_t><<<grid, 256, 0, s>>>(hxp, dp, hxa, da, hy, rows, static_cast<uint16_t*>(xp),
                                                               ld_p, static_cast<uint16_t*>(xa), ld_a, y);
    } else {
        static const bool split = shared_split(stage_rows_bits_kernel<uint32_t>);
        (void)split;
        stage_rows_bits_kernel<uint32_t><<<grid, 256, 0, s>>>(hxp, dp, hxa, da, hy, rows, static_cast<uint32_t*>(xp),
                                                               ld_p, static_cast<uint32_t*>(xa), ld_a, y);
    }
    return cudaGetLastError();
}

}  // namespace vfl
