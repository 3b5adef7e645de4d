// Fused one-launch-per-phase kernels for narrow fp32 models.
#pragma once

#include "vfl_kernels.cuh"

namespace vfl {

constexpr int kFusedThreads = 512;
constexpr int kFusedRows = 16;                 // rows per row tile
constexpr int kFusedMaxWidth = 256;            // widest layer input or output
constexpr int kFusedMaxLayers = 16;
constexpr size_t kFusedMaxSmem = 227 * 1024;

// shared-memory row stride >= width, = 4 mod 32 (the MMA A fragments and the
// forward's B fragments read 8 rows x 4 columns conflict-free), a 16-byte multiple
inline int fused_act_stride(long long width) { return (int)(((width + 27) / 32) * 32 + 4); }
inline int fused_w_stride(long long ld) { return fused_act_stride(ld); }

struct FusedLayerArgs {
    int in, out;
    long long in_ld;         // row stride of W copies
    long long out_ld;        // row stride of activations this layer writes
    const float* W;          // weight version read by this step, [out, in_ld]
    const float* b;
    int ws_off;              // shared-memory offset (floats) of W, -1 when not staged
    int ws_ld;               // its shared-memory row stride (= 4 mod 32)
    float* Y; long long ldy; // forward output rows of this step (global)
    float* D; long long ldd; // d(pre-activation) rows of this step (global), written in phase 1
    long long poff;          // offset of this layer's [W | b] gradient in the flat parameter vector
    float* Wm; float* bm;    // fp32 master (SGD)
    float* Wc; float* bc;    // copy of the new version
    float* gW; float* gb;    // reduced gradient (read back by vfl_get_grads)
};

// Passive forward of one step.
struct FusedChainArgs {
    FusedLayerArgs L[kFusedMaxLayers];
    int nl;
    const float* x; long long ldx;
    int rows, act_ld, w_floats;
    int* counter;
    ChannelHeader* hdr;
    long long k; int batch, version;
};

// Active step (L[0..na) = f_a, L[na..na+nt) = g) or passive backward (L[0..nl) = f_p).
struct FusedStepArgs {
    FusedLayerArgs L[kFusedMaxLayers];
    int na, nt;                         // passive backward: na = layers of f_p, nt = 0
    int rows, act_ld, w_floats;
    const float* x; long long ldx;      // active: x_a rows of the step; passive: x_p rows
    const int* y;                       // labels of the step's rows (active)
    int loss;
    const float* zp; long long ldzp;    // active: published embedding to read
    float* gradp; long long ldgp;       // active: gradient payload to publish; passive: to read
    float* ds;                          // active: d(logits) [rows, n_out]
    float* rowloss;                     // active: per-row loss
    float* loss_out;
    float* part; long long ptotal;      // per-row-tile partial gradients [tiles][ptotal]
    float lr;
    const ChannelHeader* chk_hdr;       // header to check (embedding / gradient channel)
    ChannelHeader* pub_hdr;             // header to publish (active: gradient channel)
    long long k; int batch, version;
    int* status;
};

// Shared memory: every staged weight matrix (w_floats, laid out by ws_off /
// wts_off) followed by row-tile activation slots of kFusedRows x act_ld.
// plus 1024 floats for the K-split partial sums of the tile GEMMs (8 tiles x 32 lanes x 4)
constexpr int kFusedRedFloats = 1024;
inline size_t fused_smem_fwd(int w_floats, int act_ld) {
    return (size_t)(w_floats + 2 * kFusedRows * act_ld + kFusedRedFloats) * sizeof(float);
}
inline size_t fused_smem_active(int w_floats, int act_ld, int na, int nt) {
    return (size_t)(w_floats + (na + nt + 4) * kFusedRows * act_ld + kFusedRedFloats) * sizeof(float);
}
inline size_t fused_smem_pbwd(int w_floats, int act_ld, int nl) {
    return (size_t)(w_floats + (nl + 3) * kFusedRows * act_ld + kFusedRedFloats) * sizeof(float);
}

cudaError_t launch_fused_passive_fwd(const FusedChainArgs& a, cudaStream_t s);
cudaError_t launch_fused_active(const FusedStepArgs& a, int grid, cudaStream_t s);
cudaError_t launch_fused_passive_bwd(const FusedStepArgs& a, int grid, cudaStream_t s);
// Largest cooperative grid of the active (which = 0) or passive-backward (1) kernel with `smem` bytes.
cudaError_t fused_max_grid(int which, size_t smem, int* ctas);

}  // namespace vfl
