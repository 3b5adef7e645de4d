// Internal declarations shared by the kernels and the host runtime of libvfl.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "vfl.h"

namespace vfl {

// Header written after a channel payload (embedding or gradient) is complete.
struct ChannelHeader {
    long long k;      // step that published the slot
    int batch;        // batch id j of that step
    int version;      // weight version that produced the payload
};

// Bits of the device status word.
enum : int { ST_VERSION = 1, ST_TIMEOUT = 2, ST_KERNEL_TIMEOUT = 4 };

enum GemmMode : int { GEMM_FWD = 0, GEMM_DX = 1, GEMM_DW = 2 };

// C[m, n] = sum_k A(m, k) * B(n, k) with strided operands.
//   A(m, k) = A[m * a_rs + k * a_cs]   (k >= ka reads A2[m * a2_rs + (k - ka) * a_cs])
//   B(n, k) = B[n * b_rs + k * b_cs]
// Epilogues:
//   FWD: C = act(acc + bias[n]); act = ReLU when relu != 0.
//   DX : columns n < n_split go to C (masked by mask1[m, n] > 0 when mask1 != 0),
//        columns n >= n_split to C2 at column n - n_split (masked by mask2 when set).
//   DW : split-K partial: P[z * p_stride + m * ldc + n] = sum over k in chunk z;
//        Pb[z * pb_stride + m] = sum_k A(m, k) over the chunk (bias gradient).
// Channel-header work folded into a kernel of the step (instead of a one-thread kernel of its own):
// thread 0 of CTA 0 checks `chk` at entry (another step's header sets ST_VERSION in *status) and writes
// `pub` = {k, batch, version} when it ends; readers of `pub` wait for the whole grid to complete first.
struct HeaderOps {
    ChannelHeader* pub;
    const ChannelHeader* chk;
    long long k;
    int batch, version;
    int* status;
};
#ifdef __CUDACC__
__device__ __forceinline__ bool first_thread_of_grid() {
    return blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0 && threadIdx.x == 0;
}
__device__ __forceinline__ void header_check(const HeaderOps& h) {
    if (h.chk && first_thread_of_grid() && h.chk->k != h.k) atomicOr(h.status, ST_VERSION);
}
__device__ __forceinline__ void header_publish(const HeaderOps& h) {
    if (h.pub && first_thread_of_grid()) {
        h.pub->k = h.k;
        h.pub->batch = h.batch;
        h.pub->version = h.version;
    }
}
#endif

struct GemmArgs {
    int mode;
    int M, N, K;
    const void* A; long long a_rs, a_cs;
    const void* A2; long long a2_rs; int ka;
    const void* B; long long b_rs, b_cs;
    const float* bias; int relu;
    void* C; long long ldc; int c_bf16;
    void* C2; long long ldc2; int c2_bf16; int n_split;
    const void* mask1; long long mask1_ld;
    const void* mask2; long long mask2_ld;
    float* P; long long p_stride;
    float* Pb; long long pb_stride;
    int kchunk;
    HeaderOps hdr;
};

// Launch the SIMT GEMM (fp32 FFMA).  a_bf16 / b_bf16 select operand element
// types; masks share the element type of the compute dtype (mask_bf16).
cudaError_t launch_gemm_simt(const GemmArgs& g, int a_bf16, int b_bf16, int mask_bf16, int nsplit,
                             cudaStream_t s);

// Loss + d(logits) over one batch (single block, deterministic reduction):
//   rows: B_k; logits fp32 [B_k, n_out]; y int32 labels of the batch rows.
//   ds [B_k, n_out] = dLoss/dlogits of the batch-mean loss; loss_out = mean loss.
// A dropped step's loss: NaN in the loss ring slot and, when given, in the host ring slot.
cudaError_t launch_mark_dropped(float* loss, float* loss_host, cudaStream_t s);
cudaError_t launch_loss(const float* logits, const int* y, int rows, int n_out, int loss_kind, float* ds,
                        float* loss_out, float* loss_host, cudaStream_t s);

// DP on the published gradient (one block per row):
//   in fp32 [rows, e] (ld_in), out compute dtype [rows, e] (ld_out).
cudaError_t launch_dp(const float* in, long long ld_in, void* out, long long ld_out, int out_bf16, int rows,
                      int e, float clip, float sigma, unsigned long long seed, long long k, cudaStream_t s);

// DP on the published embedding (one block per row): z and out in the compute dtype [rows, e] (ld),
// out = c z + sigma clip N(0,1) with c = min(1, clip / ||z||) per row, written to scale_out[rows].
cudaError_t launch_dp_emb(const void* z, long long ld, int bf16, void* out, float* scale_out, int rows, int e,
                          float clip, float sigma, unsigned long long seed, long long k, cudaStream_t s);

// out[r, c] = g[r, c] * (z[r, c] > 0), compute dtype, [rows, e] with leading dim ld; with row_scale,
// g[r, c] is first multiplied by row_scale[r] (and rounded to the compute dtype).
cudaError_t launch_relu_mask(const void* g, const void* z, void* out, long long ld, int rows, int e, int bf16,
                             const float* row_scale, const HeaderOps& hdr, cudaStream_t s);

struct SgdLayer {
    float* W; float* b;           // fp32 master
    const float* pW; const float* pb;  // split-K partial gradients
    long long pW_stride, pb_stride;
    int nsplit;                   // partials of dW
    int nsplit_b;                 // partials of db
    int out, in, in_ld;
    void* cW; float* cb;          // compute copy to write (ring slot of the new version)
    long long begin;              // first flat element index of this layer
};
constexpr int kMaxSgdLayers = 16;
struct SgdArgs {
    SgdLayer L[kMaxSgdLayers];
    int n_layers;
    long long total;
    float lr;
    int c_bf16;
};
cudaError_t launch_sgd(const SgdArgs& a, cudaStream_t s);

// Parameter-server aggregation (Sec. 4.1, Eq. 5): every replica of a party's layers takes the mean of the
// replicas, summed in fp32 in replica order and divided by nrep (IEEE division); the fp32 masters
// and the compute copies [out, in_ld] (padding columns untouched) are all rewritten.  The layer
// table lives in device memory; layer l covers flat indices [begin, begin + out * in + out).
constexpr int kPsMaxRep = 16;
struct PsAvgLayer {
    float* Wr[kPsMaxRep]; float* br[kPsMaxRep];   // fp32 masters per replica
    void* cW[kPsMaxRep]; float* cb[kPsMaxRep];    // compute copies per replica
    int out, in;
    long long in_ld;
    long long begin;
};
cudaError_t launch_ps_average(const PsAvgLayer* tab, int n_layers, long long total, int nrep, int c_bf16,
                              cudaStream_t s);

// Output layer of g (n_out <= kHeadMaxOut outputs over K <= kHeadMaxK bf16 inputs) with the loss
// folded in, for the bf16 path: per row the logits s = h W^T + b (fp32), the row's loss and
// ds = dloss/ds / B (Eq. 1 or softmax cross-entropy), and the hidden layer's d(pre-activation)
// (ds W) * [h > 0] rounded to bf16; per block of kHeadRows rows the partial dW = ds^T h and
// db = sum of ds (reduced by the SGD kernel in block order), and the step's mean loss from the
// block sums in block order (the last block to finish).
constexpr int kHeadMaxOut = 12;
constexpr int kHeadMaxK = 256;
constexpr int kHeadRows = 16;
struct HeadArgs {
    const void* h; long long ldh;     // g's last hidden activation rows [rows, ldh], bf16
    const void* W; long long ldw;     // the output layer's version copy [n_out, ldw], bf16
    const float* b;                   // its bias, fp32
    int K, nout, rows, loss;
    const int* y;
    float* logits;                    // [rows, n_out]
    float* ds;                        // [rows, n_out]
    void* dh; long long lddh;         // hidden layer's d(pre-activation) [rows, lddh], bf16
    float* pW; long long pw_stride;   // [blocks][n_out * K]
    float* pb; long long pb_stride;   // [blocks][n_out]
    int nblk;                         // blocks launched, >= head_blocks(rows); blocks past the rows write zero partials
    float* blk_loss;                  // [blocks]
    int* counter;                     // blocks finished (re-armed by the last)
    float* loss_out;
    float* loss_host;                 // a second copy of the mean loss in mapped host memory (or null)
};
inline int head_blocks(int rows) { return (rows + kHeadRows - 1) / kHeadRows; }
cudaError_t launch_head(const HeadArgs& a, cudaStream_t s);

cudaError_t launch_write_header(ChannelHeader* h, long long k, int batch, int version, cudaStream_t s);
cudaError_t launch_check_header(const ChannelHeader* h, long long k, int* status, cudaStream_t s);
cudaError_t launch_wait_header(const ChannelHeader* h, long long k, long long max_iters, int* status,
                               cudaStream_t s);
cudaError_t launch_cast_rows(const float* src, int rows, int d, void* dst, long long ld, int bf16, cudaStream_t s);
// Stage one step's rows from host-resident (mapped) arrays: x_p [rows, dp] and x_a [rows, da] fp32 into
// rows of ld_p / ld_a elements (bf16 or fp32, padding columns zero), and the labels.
cudaError_t launch_stage_rows(const float* hxp, int dp, const float* hxa, int da, const int* hy, int rows, void* xp,
                              long long ld_p, void* xa, long long ld_a, int* y, int bf16, cudaStream_t s);
// The same for bf16 host rows into a bf16 context (no rounding: a 16-byte copy of eight elements per thread).
cudaError_t launch_stage_rows_b16(const uint16_t* hxp, int dp, const uint16_t* hxa, int da, const int* hy, int rows,
                                  void* xp, long long ld_p, void* xa, long long ld_a, int* y, cudaStream_t s);
// The same for bit-packed binary host rows (ceil(d / 32) words a row, feature c in bit c mod 32 of word c / 32)
// into bf16 (bf16 != 0) or fp32 slot rows of 0 / 1 values.
cudaError_t launch_stage_rows_bits(const uint32_t* hxp, int dp, const uint32_t* hxa, int da, const int* hy, int rows,
                                   void* xp, long long ld_p, void* xa, long long ld_a, int* y, int bf16,
                                   cudaStream_t s);
// Sets the message vfl_last_error(NULL) returns on this thread.
void set_global_error(const char* msg);

cudaError_t launch_to_f32(const void* src, long long ld, int rows, int cols, int bf16, float* dst, cudaStream_t s);

}  // namespace vfl
