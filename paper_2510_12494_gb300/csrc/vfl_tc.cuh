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
//  DW : P[M=out, N=in] = A[rows, out]^T B[rows, in] (row stride ldc), reduced over
//       the batch inside a thread-block cluster (partials through `ws`); B may be [B | B2] split at column
//       kb; Pb[out] = column sums of A (when Pb is set).  With Wm set, the SGD step
//       of Eq. 2 follows in the same kernel: Wm -= lr P, bm -= lr Pb (fp32
//       masters), cW [out, cw_ld] = bf16(Wm) and cb = bm (the new version's copies).
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
    float* P;
    float* Pb;
    float* ws; long long ws_floats;   // DW: partial-tile exchange (tc_dw_ws_floats(M, N, K) floats)
    float* Wm; float* bm;       // DW with the SGD step: fp32 masters (null: gradient only)
    void* cW; long long cw_ld;  // the new version's bf16 copy of W
    float* cb;                  // and of b
    float lr;
    int* err;                   // status word: ST_KERNEL_TIMEOUT when a bounded wait gave up
    HeaderOps hdr;              // channel header checked at entry / published at the end (or none)
};

// The driver's tensor-map encoder is reachable (false on machines without a driver).
bool tc_available();
// Split-K factor and chunk of a tensor-core weight gradient over `rows` as the workspace sees it:
// one reduced gradient (the cluster reduces its ranks' partials on chip).
void tc_choose_split(int out, int in, int rows, int* nsplit, int* kchunk);
// Tensor-core weight gradient: the workspace (floats) its partial tiles go through for a batch of `rows`
// (enough for every plan tc_dw_plan can pick), and its tile width and cluster size.
long long tc_dw_ws_floats(int out, int in, int rows);
void tc_dw_plan(int out, int in, int rows, bool concat, int kb, long long ws_floats, int* bn, int* cs);
// Shape rule for the tensor-core weight gradient (independent of the driver).
bool tc_shape_dw(int out, int in, bool concat, int kb);
bool tc_supported_fwd(int in, int out, bool concat, int ka, bool out_f32);
bool tc_supported_dx(int in, int out, int n_split, bool c2_f32);
bool tc_supported_dw(int out, int in, bool concat, int kb);
cudaError_t launch_tc_gemm(const TcGemm& g, cudaStream_t s);

// A bottom model's whole forward for every 128-row tile in one launch (each layer 128 or 256 wide, 2-4
// layers, the first layer's input at most 256 wide): Y_l = relu(Y_{l-1} W_l^T + b_l), Y_{-1} = X [M, ldx];
// W_l [out_l, ldw_l] and every Y_l [M, ldy_l] bf16, biases fp32.  The activations stay in shared memory
// between layers; every Y_l is also written out.  The header ops are those of the last layer's output.
struct TcChain {
    int L, M, K0;
    const void* X; long long ldx;
    const void* W[4]; long long ldw[4];
    int out[4];
    const float* bias[4];
    void* Y[4]; long long ldy[4];
    int* err;
    HeaderOps hdr;
};
bool tc_chain_supported(int L, int K0, const int* out);
cudaError_t launch_tc_chain(const TcChain& c, cudaStream_t s);

}  // namespace vfl
