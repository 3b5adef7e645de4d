// Fused one-launch-per-phase kernels for narrow fp32 models.
#pragma once

#include "vfl_kernels.cuh"

namespace vfl {

constexpr int kFusedThreads = 512;
constexpr int kFusedRows = 16;                 // rows per row tile
constexpr int kFusedMaxWidth = 256;            // widest layer input or output
constexpr int kFusedMaxLayers = 16;
constexpr int kFusedMaxOut = 16;               // n_out up to which the output layer is folded into an epilogue
constexpr size_t kFusedMaxSmem = 227 * 1024;

// shared-memory row stride >= width, = 4 mod 32 (the MMA A fragments and the
// forward's B fragments read 8 rows x 4 columns conflict-free), a 16-byte multiple
inline int fused_act_stride(long long width) { return (int)(((width + 27) / 32) * 32 + 4); }
inline int fused_w_stride(long long ld) { return fused_act_stride(ld); }
// shared-memory floats of a staged layer: W in ceil8(out) rows of fused_w_stride, then b over ceil8(out)
inline long long fused_layer_floats(int out, long long in_ld) {
    const long long out8 = (out + 7) / 8 * 8;
    return out8 * fused_w_stride(in_ld) + out8;
}

// Warp mapping of a 16-row tile GEMM with ks k-steps and ntl output blocks of 8
// columns (kFusedThreads = 512, 16 warps): 2^lng warps cover the blocks, up to
// 4 each (tpw), and 2^lkg groups of them split the k-steps, as many as fit the
// 16 warps, the k-steps and the partial buffer (16 rows x (8 ntl + 8) floats
// per group).  Packed as lng | lkg << 4 | tpw << 8.
constexpr int kFusedRedFloats = 8192;
inline __host__ __device__ int fused_gemm_map(int ks, int ntl) {
    const int lng = ntl <= 4 ? 0 : ntl <= 8 ? 1 : ntl <= 16 ? 2 : 3;
    const int tpw = (ntl + (1 << lng) - 1) >> lng;
    int lkg = 4 - lng;
    while (lkg > 0 && ((1 << lkg) > ks || ((16 * (8 * ntl + 8)) << lkg) > kFusedRedFloats)) --lkg;
    return lng | lkg << 4 | tpw << 8;
}

struct FusedLayerArgs {
    int in, out;
    int fmap, dmap;          // fused_gemm_map of the forward and of the input-gradient GEMM
    long long in_ld;         // row stride of W copies
    long long out_ld;        // row stride of activations this layer writes
    const float* W;          // weight version read by this step, [out, in_ld]
    const float* b;
    int ws_off;              // shared-memory offset (floats) of W, -1 when not staged
    int ws_ld;               // its shared-memory row stride (= 4 mod 32)
    float* Y; long long ldy; // forward output rows of this step (global)
    float* D; long long ldd; // d(pre-activation) rows of this step (global)
};

// Passive forward of one step.
struct FusedChainArgs {
    FusedLayerArgs L[kFusedMaxLayers];
    int nl;
    const float* x; long long ldx;
    int rows, act_ld, w_floats;
    ChannelHeader* hdr;
    long long k; int batch, version;
    // DP on the published embedding (App. C), when dp_out is set: per row c = min(1, C / ||z||), the
    // payload c z + sigma C N(0,1) (Philox tag 0x4445) to dp_out, c to dp_scale
    float* dp_out; long long ld_dp;
    float* dp_scale;
    float dp_clip, dp_sigma;
    unsigned long long dp_seed;
};

// Row-parallel part of the active step (L[0..na) = f_a, L[na..na+nt) = g) or of
// the passive backward (L[0..na) = f_p, nt = 0): forward and input-gradient
// chains, one 16-row tile per CTA; the weight gradients come from the update kernel.
struct FusedStepArgs {
    FusedLayerArgs L[kFusedMaxLayers];
    int na, nt;
    int rows, act_ld, w_floats;
    const float* x; long long ldx;      // active: x_a rows of the step
    const int* y;                       // labels of the step's rows (active)
    int loss;
    const float* zp; long long ldzp;    // active: published embedding to read
    float* zpc; long long ldzpc;        // active: copy of z^p kept for the weight gradient of g's first layer
    float* gradp; long long ldgp;       // active: gradient payload to publish; passive: to read
    float* rowloss;                     // active: per-row loss
    const ChannelHeader* chk_hdr;       // header to check (embedding / gradient channel)
    ChannelHeader* pub_hdr;             // header to publish (active: gradient channel)
    long long k; int batch, version;
    int* status;
    const float* rowscale;              // passive, DP on the embedding: the rows' clip factors (else null)
};

// Weight gradient + SGD of a set of layers: dW = D^T X and db = column sums of D
// over the step's rows, then Eq. 2 on the master and the new version's copy.
constexpr int kUpdThreads = 256;
constexpr int kUpdCluster = 8;        // CTAs per output tile, each over 1/8 of the rows
constexpr int kUpdTile = 32;          // output tile: 32 outputs x 32 inputs
struct FusedUpdLayer {
    int out, in;
    long long in_ld;                  // row stride of the version copy
    const float* D; long long ldd;    // d(pre-activation) rows [rows, out]
    const float* X; long long ldx;    // input columns [0, xsplit)
    const float* X2; long long ldx2;  // input columns [xsplit, in), indexed from 0
    int xsplit;
    int x_early;                      // X is not written by the grid this launch depends on programmatically
    int tile0, tiles_i;               // first output tile of this layer, tiles along the input
    float* Wm; float* bm;             // fp32 master
    float* Wc; float* bc;             // the new version's copy
    float* gW; float* gb;             // the reduced gradient (read back by vfl_get_grads)
};
struct FusedUpdArgs {
    FusedUpdLayer L[kFusedMaxLayers];
    int nl, ntiles, rows;
    float lr;
    const float* rowloss;             // mean loss of the step from these (nullptr: none)
    float* loss_out;
    float* loss_host;                 // a second copy of it in mapped host memory (nullptr: none)
};
// Fills the tile bookkeeping of L[0..nl) and returns the number of output tiles.
inline int fused_update_tiles(FusedUpdLayer* L, int nl) {
    int t = 0;
    for (int l = 0; l < nl; ++l) {
        L[l].tile0 = t;
        L[l].tiles_i = (L[l].in + kUpdTile - 1) / kUpdTile;
        t += L[l].tiles_i * ((L[l].out + kUpdTile - 1) / kUpdTile);
    }
    return t;
}

// Shared memory: every staged weight matrix (w_floats, laid out by ws_off),
// then fp32 row tiles of kFusedRows x act_ld floats, then kFusedRedFloats for
// the partial output blocks of the tile GEMMs.
// passive forward: x_p rows and a ping-pong pair
inline size_t fused_smem_fwd(int w_floats, int act_ld) {
    return (size_t)(w_floats + 3 * kFusedRows * act_ld + kFusedRedFloats) * sizeof(float);
}
// active step: x_a rows (later the logits), f_a's hidden outputs, [z^a | z^p],
// g's hidden outputs, two gradients
inline size_t fused_smem_active(int w_floats, int act_ld, int na, int nt) {
    return (size_t)(w_floats + (na + nt + 2) * kFusedRows * act_ld + kFusedRedFloats) * sizeof(float);
}
// passive backward: f_p's saved outputs, dz^p rows, two gradients
inline size_t fused_smem_pbwd(int w_floats, int act_ld, int nl) {
    return (size_t)(w_floats + (nl + 3) * kFusedRows * act_ld + kFusedRedFloats) * sizeof(float);
}

// Programmatic dependent launch outside CUDA graphs (a captured graph gets the same dependencies as
// programmatic edges instead).  serialize: the kernel may launch once the previous kernel on its
// stream has triggered (it waits for that grid before reading its output).  pevent: an event recorded
// by the launch that fires once every CTA of this kernel has triggered; a kernel on another stream
// that waits on it may launch then and waits for this grid before reading its output.
struct LaunchOpt {
    int serialize = 0;
    cudaEvent_t pevent = nullptr;
};

cudaError_t launch_fused_passive_fwd(const FusedChainArgs& a, cudaStream_t s, const LaunchOpt& o = LaunchOpt());
cudaError_t launch_fused_active(const FusedStepArgs& a, cudaStream_t s, const LaunchOpt& o = LaunchOpt());
cudaError_t launch_fused_passive_bwd(const FusedStepArgs& a, cudaStream_t s, const LaunchOpt& o = LaunchOpt());
cudaError_t launch_fused_update(const FusedUpdArgs& a, cudaStream_t s, const LaunchOpt& o = LaunchOpt());

// Whether a kernel (its function pointer, as a graph kernel node records it) is one of the fused kernels
// above, which place their programmatic waits themselves; every other kernel of the library waits at entry.
bool is_fused_kernel(const void* func);

}  // namespace vfl
