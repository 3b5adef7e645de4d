// Tensor-core (tcgen05 + TMEM + TMA) GEMMs for the bf16 layers of the step.
#pragma once

#include <cuda_runtime.h>

#include "vfl_kernels.cuh"

namespace vfl {

// One Linear-layer GEMM on bf16 operands with fp32 accumulation in TMEM.
//  FWD: C[M=rows, N=out] = act(A[rows, K=in] W^T + bias); A may be [A | A2]
//       split at column ka; B = W [out, ldb]; C bf16 (ldc).
//  DX : C[rows, N=in] = A[rows, K=out] W, B = W [out, ldb] (MN-major operand);
//       columns < n_split -> C masked by mask1 > 0; the rest -> C2 (bf16),
//       masked by mask2 when given.
//  DW : P[z][M=out, N=in] = sum over rows of chunk z of A[rows, out]^T B[rows, in]
//       (both MN-major operands), B may be [B | B2] split at column kb;
//       Pb[z][out] = column sums of A over the chunk.
struct TcGemm {
    int mode;
    int M, N, K;
    const void* A; long long lda;
    const void* A2; long long lda2; int ka;
    const void* B; long long ldb;
    const void* B2; long long ldb2; int kb;
    const float* bias; int relu;
    void* C; long long ldc;
    const void* mask1;
    int n_split;
    void* C2; long long ldc2;
    const void* mask2;
    int c2_f32;                 // DX: C2 is fp32 (the DP path perturbs it before publishing)
    float* P; long long p_stride;
    float* Pb; long long pb_stride;
    int nsplit, kchunk;
    int* err;                   // status word: ST_KERNEL_TIMEOUT when a bounded wait gave up
    HeaderOps hdr;              // channel header checked at entry / published at the end (or none)
};

// The driver's tensor-map encoder is reachable (false on machines without a driver).
bool tc_available();
// Split-K factor and chunk (a multiple of 64 rows) of a tensor-core weight gradient over `rows`.
void tc_choose_split(int out, int in, int rows, int* nsplit, int* kchunk);
// Shape rule for the tensor-core weight gradient (independent of the driver).
bool tc_shape_dw(int out, int in, bool concat, int kb);
bool tc_supported_fwd(int in, int out, bool concat, int ka, bool out_f32);
bool tc_supported_dx(int in, int out, int n_split, bool c2_f32);
bool tc_supported_dw(int out, int in, bool concat, int kb);
cudaError_t launch_tc_gemm(const TcGemm& g, cudaStream_t s);

}  // namespace vfl
