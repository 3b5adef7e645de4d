// Fused kernels for narrow fp32 models (every width <= 256): each phase of
// Algorithm 1 is one row-parallel launch, and each party's weight gradient and
// SGD step (Eq. 2, delayed form of App. D) is one more.
//
//  - passive forward: every CTA stages all of f_p's weights into shared memory
//    with cp.async, then runs the bottom chain for its 16-row tile; CTA 0 writes
//    the embedding channel's header.
//  - active step: active bottom forward, top forward on [z^a | z^p], loss, the
//    input-gradient chain back to the first active layer; dz^p goes to the
//    gradient channel (header written by CTA 0), every layer's
//    d(pre-activation) rows stay in HBM for the update.
//  - passive backward: the input-gradient chain of f_p from dz^p.
//  - update (one per party): dW = D^T X over the step's rows for every layer,
//    an output tile per cluster of 8 CTAs that each take 1/8 of the rows; each
//    CTA pushes its partial of the outputs another rank owns into that rank's
//    shared memory, the owners sum the 8 partials in rank order (deterministic)
//    and SGD writes the master and the new version's copy.
//
// The row-tile GEMMs run on the warp-level tensor cores (mma.sync m16n8k8,
// TF32) in 3xTF32 form, which keeps fp32 accuracy: x = hi + lo with hi, lo
// TF32, and a b ~ a_hi b_hi + a_lo b_hi + a_hi b_lo.  Activation tiles live in
// shared memory in fp32; their A fragments are loaded with ldmatrix and split
// in registers, and weights are split as they are read.  Every tile is
// zero-padded to a multiple of 8 columns and
// every staged weight matrix to a multiple of 8 rows, so the GEMM loops need no
// bounds checks.
#include <cooperative_groups.h>

#include "vfl_fused.cuh"
#include "vfl_philox.cuh"

namespace cg = cooperative_groups;

namespace vfl {

namespace {

constexpr int NT = kFusedThreads;     // 16 warps

// Programmatic dependent launch.  Inside a graph whose edge into this kernel is
// programmatic, the kernel may start while its producer still runs:
// griddep_wait() returns once the producer grid has completed and its writes
// are visible, so every read of the producer's output comes after it.
// griddep_trigger() lets this kernel's own programmatic dependents launch.
// Without such edges both are no-ops.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
constexpr int NW = NT / 32;
constexpr int R = kFusedRows;
static_assert(R == 16, "the MMA tiles cover exactly 16 rows");
static_assert(NW == R, "row-tile copies give each warp one row");

__device__ __forceinline__ int ceil8(int x) { return (x + 7) & ~7; }

// The channel header of a published payload, written by CTA 0.  Every subscriber is ordered after
// the publishing kernel's completion (stream order, an event, or a programmatic dependency whose
// wait returns once the grid has completed), which makes all of the grid's payload writes visible
// with the header; so no CTA needs to wait for the others or fence its writes here.
__device__ __forceinline__ void publish_header(ChannelHeader* hdr, long long k, int batch, int version) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        hdr->k = k;
        hdr->batch = batch;
        hdr->version = version;
    }
}

__device__ __forceinline__ void cp16(float* s, const float* g) {
    const unsigned sa = (unsigned)__cvta_generic_to_shared(s);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(sa), "l"(g) : "memory");
}

// 4 bytes, or zero-fill when !valid (src must still be a valid address)
__device__ __forceinline__ void cp4(float* s, const float* g, bool valid) {
    const unsigned sa = (unsigned)__cvta_generic_to_shared(s);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(sa), "l"(g), "r"(valid ? 4 : 0) : "memory");
}

__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }

// wait until at most n committed groups are still in flight (n <= 8), then make them visible block-wide
__device__ __forceinline__ void cp_wait_pending(int n) {
    switch (n) {
        case 0: asm volatile("cp.async.wait_group 0;\n" ::: "memory"); break;
        case 1: asm volatile("cp.async.wait_group 1;\n" ::: "memory"); break;
        case 2: asm volatile("cp.async.wait_group 2;\n" ::: "memory"); break;
        case 3: asm volatile("cp.async.wait_group 3;\n" ::: "memory"); break;
        case 4: asm volatile("cp.async.wait_group 4;\n" ::: "memory"); break;
        case 5: asm volatile("cp.async.wait_group 5;\n" ::: "memory"); break;
        case 6: asm volatile("cp.async.wait_group 6;\n" ::: "memory"); break;
        case 7: asm volatile("cp.async.wait_group 7;\n" ::: "memory"); break;
        default: asm volatile("cp.async.wait_group 8;\n" ::: "memory"); break;
    }
    __syncthreads();
}

// R rows of `cols` floats (cols % 4 == 0): rows < nrows copied asynchronously
// from global (row stride ldg), the rest zero-filled; smem row stride lds.
// Warp r copies row r.
__device__ void async_rows(float* s, int lds, const float* g, long long ldg, int cols, int nrows) {
    const int r = threadIdx.x >> 5;
    for (int c = (threadIdx.x & 31) * 4; c < cols; c += 128) {
        if (r < nrows)
            cp16(s + r * lds + c, g + (long long)r * ldg + c);
        else
            *reinterpret_cast<float4*>(s + r * lds + c) = make_float4(0.f, 0.f, 0.f, 0.f);
    }
}

// rows x cols floats (cols % 4 == 0, 16-byte aligned rows) into smem rows of stride lds, asynchronously.
// A source whose rows are contiguous (ldg == cols) with a power-of-two number of 16-byte chunks per row
// is walked chunk by chunk over all lanes (narrow rows would otherwise leave most lanes of each
// copy instruction idle, and the copies cost per instruction, not per byte).
__device__ void async_matrix(float* s, int lds, const float* g, long long ldg, int rows, int cols) {
    const int q = cols >> 2;
    if (ldg == cols && (q & (q - 1)) == 0) {
        const int lq = __ffs(q) - 1;
        for (int i = threadIdx.x; i < rows * q; i += NT) {
            const int r = i >> lq, c = (i & (q - 1)) << 2;
            cp16(s + r * lds + c, g + (long long)r * ldg + c);
        }
        return;
    }
    for (int r = threadIdx.x >> 5; r < rows; r += NW)
        for (int c = (threadIdx.x & 31) * 4; c < cols; c += 128) cp16(s + r * lds + c, g + (long long)r * ldg + c);
}

// A staged layer, asynchronously: W's rows (stride ws_ld), zero rows up to
// ceil8(out), then b over ceil8(out) floats, zero past out.  The version copies keep their
// columns [in, in_ld) zero, so every staged tile is zero-padded both ways.
__device__ void stage_layer_weights(float* ws, const FusedLayerArgs& L) {
    if (L.ws_off < 0) return;
    float* w = ws + L.ws_off;
    async_matrix(w, L.ws_ld, L.W, L.in_ld, L.out, (int)L.in_ld);
    const int out8 = ceil8(L.out);
    for (int r = L.out + (threadIdx.x >> 5); r < out8; r += NW)
        for (int c = (threadIdx.x & 31) * 4; c < L.in_ld; c += 128)
            *reinterpret_cast<float4*>(w + r * L.ws_ld + c) = make_float4(0.f, 0.f, 0.f, 0.f);
    float* b = w + out8 * L.ws_ld;
    for (int c = threadIdx.x; c < out8; c += NT) cp4(b + c, L.b + (c < L.out ? c : 0), c < L.out);
}

__device__ __forceinline__ const float* staged_bias(const float* ws, const FusedLayerArgs& L) {
    return ws + L.ws_off + ceil8(L.out) * L.ws_ld;
}

// ---- 3xTF32 on mma.sync m16n8k8 ---------------------------------------------
// TF32 rounding to nearest, ties away from zero, on the bit pattern: adding half
// an ulp of the 10-bit mantissa to the magnitude bits carries into the exponent
// exactly when rounding up crosses a binade.
__device__ __forceinline__ uint32_t to_tf32(float x) { return (__float_as_uint(x) + 0x1000u) & 0xffffe000u; }

__device__ __forceinline__ void split_tf32(float x, uint32_t& hi, uint32_t& lo) {
    hi = to_tf32(x);
    lo = to_tf32(x - __uint_as_float(hi));
}

// d += a b (m16n8k8, TF32 inputs, fp32 accumulation); no side effects, so the
// compiler may interleave independent MMAs
__device__ __forceinline__ void mma_tf32(float* d, const uint32_t* a, const uint32_t* b) {
    asm("mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// A fragment (fp32 bits) of a 16 x 8 block of a 16-row tile: ldmatrix of four
// 8 x 4 (32-bit) matrices, rows 0-7 / 8-15 by columns k0..k0+3 / k0+4..k0+7.
// Lane l points at row (l mod 8) + 8 ((l / 8) mod 2), column k0 + 4 (l / 16)
// (a16_lane_offset); a row stride of 4 mod 32 floats makes it conflict-free.
__device__ __forceinline__ int a16_lane_offset(int ld) {
    const int lane = threadIdx.x & 31;
    return ((lane & 7) + ((lane >> 3) & 1) * 8) * ld + (lane >> 4) * 4;
}

__device__ __forceinline__ void lds_a(uint32_t* a, const float* p) {
    const unsigned addr = (unsigned)__cvta_generic_to_shared(p);
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3])
                 : "r"(addr));
}

constexpr int kTilesPerWarp = 4;

// For the nt <= 4 output blocks at columns 8 j0, 8 (j0 + 1), ...:
// d += A_lo B_hi + A_hi B_lo + A_hi B_hi (small terms first) over k-steps
// [ks0, ks1).  Forward (kT = false): B[k][n] = W[n][k]; input gradient
// (kT = true): B[k][n] = W[k][n]; W in smem, row stride ldw.  One A fragment
// serves all the warp's blocks, whose MMA chains are independent; the next
// k-step's operands are loaded before this one's MMAs issue.
template <bool kT>
__device__ __forceinline__ void mma_steps(float (*d)[4], const float* A, int lda, const float* W, int ldw, int j0,
                                          int nt, int ks0, int ks1) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const float* wb = kT ? W + t * ldw + j0 * 8 + g : W + (j0 * 8 + g) * ldw + t;
    const int jstep = kT ? 8 : 8 * ldw;
    const int kstep = kT ? 8 * ldw : 8;
    const int khalf = kT ? 4 * ldw : 4;
    const float* ab = A + a16_lane_offset(lda);
    uint32_t a[4];
    float b[kTilesPerWarp][2];
    auto load = [&](int ks) {
        lds_a(a, ab + ks * 8);
#pragma unroll
        for (int i = 0; i < kTilesPerWarp; ++i)
            if (i < nt) {
                const float* w = wb + i * jstep + ks * kstep;
                b[i][0] = w[0];
                b[i][1] = w[khalf];
            }
    };
    if (ks0 < ks1) load(ks0);
    for (int ks = ks0; ks < ks1; ++ks) {
        uint32_t ah[4], al[4], bh[kTilesPerWarp][2], bl[kTilesPerWarp][2];
#pragma unroll
        for (int i = 0; i < 4; ++i) split_tf32(__uint_as_float(a[i]), ah[i], al[i]);
#pragma unroll
        for (int i = 0; i < kTilesPerWarp; ++i)
            if (i < nt) {
                split_tf32(b[i][0], bh[i][0], bl[i][0]);
                split_tf32(b[i][1], bh[i][1], bl[i][1]);
            }
        if (ks + 1 < ks1) load(ks + 1);
#pragma unroll
        for (int i = 0; i < kTilesPerWarp; ++i)
            if (i < nt) mma_tf32(d[i], al, bh[i]);
#pragma unroll
        for (int i = 0; i < kTilesPerWarp; ++i)
            if (i < nt) mma_tf32(d[i], ah, bl[i]);
#pragma unroll
        for (int i = 0; i < kTilesPerWarp; ++i)
            if (i < nt) mma_tf32(d[i], ah, bh[i]);
    }
}

// C[16 x 8 ntl] = A[16 x 8 ks] B with the warp mapping `map` (fused_gemm_map):
// each group of 2^lng warps writes its 16 x 8 ntl partial, row-major (row
// stride 8 ntl + 8), to `red`; then warp r sums row r's partials in group
// order and calls epi(r, c, v0, v1) for each column pair c, c+1.  Callers put
// a barrier before each call.
static_assert(NW == 16 && R == 16, "the warp mapping assumes 16 warps and 16 rows");
// The MMA part, out of line (one copy per B layout, with its own registers).
template <bool kT>
__device__ __noinline__ void gemm_partials(const float* A, int lda, int ks, const float* W, int ldw, int ntl, int map,
                                           float* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, g = lane >> 2, t = lane & 3;
    const int lng = map & 15, lkg = (map >> 4) & 15, tpw = map >> 8;
    const int rs = 8 * ntl + 8;
    const int grp = warp >> lng, j0 = (warp & ((1 << lng) - 1)) * tpw;
    if (grp < (1 << lkg) && j0 < ntl) {
        const int nt = min(tpw, ntl - j0);
        float d[kTilesPerWarp][4] = {};
        mma_steps<kT>(d, A, lda, W, ldw, j0, nt, (grp * ks) >> lkg, ((grp + 1) * ks) >> lkg);
        float* pr = red + grp * 16 * rs + g * rs + j0 * 8 + 2 * t;
#pragma unroll
        for (int i = 0; i < kTilesPerWarp; ++i)
            if (i < nt) {
                *reinterpret_cast<float2*>(pr + i * 8) = make_float2(d[i][0], d[i][1]);
                *reinterpret_cast<float2*>(pr + 8 * rs + i * 8) = make_float2(d[i][2], d[i][3]);
            }
    }
}

template <bool kT, typename Epi>
__device__ __forceinline__ void tile_gemm(const float* A, int lda, int ks, const float* W, int ldw, int ntl, int map,
                                          float* red, Epi epi) {
    gemm_partials<kT>(A, lda, ks, W, ldw, ntl, map, red);
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const int rs = 8 * ntl + 8;
    const int r = threadIdx.x >> 5, kg = 1 << ((map >> 4) & 15);
    for (int c = 2 * lane; c < 8 * ntl; c += 64) {
        const float* src = red + r * rs + c;
        float2 v = *reinterpret_cast<const float2*>(src);
#pragma unroll 4
        for (int q = 1; q < kg; ++q) {
            const float2 u = *reinterpret_cast<const float2*>(src + q * 16 * rs);
            v.x += u.x;
            v.y += u.y;
        }
        epi(r, c, v.x, v.y);
    }
}

// Hidden-layer forward: Y = ReLU(X W^T + b) -> smem tile `out`, and to global
// rows < nrows (row stride ldyg >= ceil8(N)) when yg is set.
__device__ __forceinline__ void tile_fwd(const float* X, int ld, int K, const float* ws, int ldw, const float* bias,
                                         int N, int map, float* out, float* yg, long long ldyg, int nrows, float* red) {
    tile_gemm<false>(X, ld, ceil8(K) / 8, ws, ldw, ceil8(N) / 8, map, red, [&](int r, int c, float v0, float v1) {
        const float2 y = make_float2(fmaxf(v0 + bias[c], 0.f), fmaxf(v1 + bias[c + 1], 0.f));
        *reinterpret_cast<float2*>(out + r * ld + c) = y;
        if (yg && r < nrows) *reinterpret_cast<float2*>(yg + (long long)r * ldyg + c) = y;
    });
}

// Input gradient of a hidden layer: dX = (dY W) * [prev > 0] -> smem tile `out`
// and global rows < nrows.
__device__ __forceinline__ void tile_dx(const float* dY, int ld, int K, const float* ws, int ldw, int N, int map,
                                        const float* prev, float* out, float* og, long long ldog, int nrows,
                                        float* red) {
    tile_gemm<true>(dY, ld, ceil8(K) / 8, ws, ldw, ceil8(N) / 8, map, red, [&](int r, int c, float v0, float v1) {
        const float2 m = *reinterpret_cast<const float2*>(prev + r * ld + c);
        const float2 v = make_float2(m.x > 0.f ? v0 : 0.f, m.y > 0.f ? v1 : 0.f);
        *reinterpret_cast<float2*>(out + r * ld + c) = v;
        if (og && r < nrows) *reinterpret_cast<float2*>(og + (long long)r * ldog + c) = v;
    });
}

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(NT, 1) fused_passive_fwd_kernel(const FusedChainArgs a) {
    extern __shared__ __align__(16) float smem[];
    griddep_trigger();   // the active step may start staging its weights and rows now
    const int ld = a.act_ld;
    float* ws = smem;
    float* t0 = smem + a.w_floats;                      // x_p rows, then ping-pong
    float* t1 = t0 + R * ld;
    float* t2 = t1 + R * ld;
    float* red = t2 + R * ld;                           // partial output blocks
    const int ntiles = (a.rows + R - 1) / R;
    // one 16-row tile per CTA (the launch has one CTA per tile)
    if ((int)blockIdx.x >= ntiles) {
        griddep_wait();
        return;
    }
    {
        const int r0 = blockIdx.x * R;
        const int nr = min(R, a.rows - r0);
        async_rows(t0, ld, a.x + (long long)r0 * a.ldx, a.ldx, (int)a.L[0].in_ld, nr);
        // the weight version comes from an earlier update, which may still be finishing
        griddep_wait();
        // group l holds layer l's weights (group 0 also the rows), so layer l
        // only waits for its own weights while the later ones are still arriving
        for (int l = 0; l < a.nl; ++l) {
            stage_layer_weights(ws, a.L[l]);
            cp_commit();
        }
        const float* cur = t0;
        for (int l = 0; l < a.nl; ++l) {
            const FusedLayerArgs& L = a.L[l];
            cp_wait_pending(a.nl - 1 - l);
            float* nxt = (l & 1) ? t2 : t1;
            tile_fwd(cur, ld, L.in, ws + L.ws_off, L.ws_ld, staged_bias(ws, L), L.out, L.fmap, nxt,
                     L.Y + (long long)r0 * L.ldy, L.ldy, nr, red);
            cur = nxt;
        }
        if (a.dp_out) {
            // DP on the published embedding: warp r takes row r of the tile (the clean z stays in L.Y)
            __syncthreads();
            const int r = threadIdx.x >> 5, lane = threadIdx.x & 31;
            const int e = a.L[a.nl - 1].out;
            if (r < nr) {
                const float* zr = cur + r * ld;
                float ss = 0.f;
                for (int c = lane; c < e; c += 32) ss = fmaf(zr[c], zr[c], ss);
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
                const float norm = sqrtf(ss);
                const float f = norm > a.dp_clip ? a.dp_clip / norm : 1.0f;
                if (lane == 0) a.dp_scale[r0 + r] = f;
                const float noise = a.dp_sigma * a.dp_clip;
                const uint2 key = make_uint2((unsigned)(a.dp_seed & 0xFFFFFFFFull), (unsigned)(a.dp_seed >> 32));
                float* out = a.dp_out + (long long)(r0 + r) * a.ld_dp;
                for (int q = lane; 4 * q < e; q += 32) {
                    float xi[4] = {0.f, 0.f, 0.f, 0.f};
                    if (noise != 0.f) dp_normals4(q, r0 + r, a.k, 0x4445u, key, xi);
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        if (4 * q + j < e) out[4 * q + j] = fmaf(zr[4 * q + j], f, noise * xi[j]);
                }
            }
        }
    }
    publish_header(a.hdr, a.k, a.batch, a.version);
}

// Loss of one row (Eq. 1 in the stable logit form, or softmax cross-entropy)
// from its n_out logits s; writes d(logits) = dloss/ds / B to d.
__device__ __forceinline__ float loss_row(const float* s, int nout, int y, int loss, float inv_b, float* d) {
    if (loss == VFL_LOSS_BCE) {
        const float x = s[0];
        d[0] = (1.0f / (1.0f + expf(-x)) - (float)y) * inv_b;
        return fmaxf(x, 0.f) - x * (float)y + log1pf(expf(-fabsf(x)));
    }
    float m = s[0];
    for (int j = 1; j < nout; ++j) m = fmaxf(m, s[j]);
    float z = 0.f;
    for (int j = 0; j < nout; ++j) z += expf(s[j] - m);
    const float iz = 1.0f / z;
    for (int j = 0; j < nout; ++j) d[j] = (expf(s[j] - m) * iz - (j == y ? 1.f : 0.f)) * inv_b;
    return logf(z) + m - s[y];
}

// g's last hidden layer Lh (input X) with the output layer Lo (n_out <= MO <= kFusedMaxOut;
// MO = 1 for the BCE logit, so the per-output loops carry no predicated-off work),
// the loss and its gradient folded into the epilogue, warp r for row r:
// h = ReLU(X Wh^T + bh) -> smem tile `hs` and Lh.Y; s = h Wo^T + bo (fp32 dot
// products, reduced across the warp) -> Lo.Y; the row's loss -> rowloss;
// ds = dloss/ds / B -> Lo.D; dh = (ds Wo) * [h > 0] -> smem tile `gs` and Lh.D.
// The layers' fields come as scalars (Lh: hidden, Lo: output): a struct
// reference into kernel parameters would be copied to local memory per call.
struct TopLast {
    int h_in, h_out, h_map, h_ws_off, h_ws_ld;
    int o_out, o_ws_off, o_ws_ld;
    float* h_y; long long h_ldy;
    float* h_d; long long h_ldd;
    float* o_y; long long o_ldy;
    float* o_d; long long o_ldd;
};

template <int MO>
__device__ __noinline__ void top_last_fused(const float* X, int ld, const float* ws, TopLast L, float* hs, float* gs,
                                            const int* y, int loss, float inv_b, float* rowloss, int r0, int nr,
                                            float* red) {
    const int ntl = ceil8(L.h_out) / 8;
    gemm_partials<false>(X, ld, ceil8(L.h_in) / 8, ws + L.h_ws_off, L.h_ws_ld, ntl, L.h_map, red);
    __syncthreads();
    const int lane = threadIdx.x & 31, r = threadIdx.x >> 5;
    const int rs = 8 * ntl + 8, kg = 1 << ((L.h_map >> 4) & 15);
    const int nout = L.o_out;
    const float* bh = ws + L.h_ws_off + ceil8(L.h_out) * L.h_ws_ld;
    const float* wo = ws + L.o_ws_off;
    const int ldo = L.o_ws_ld;
    const bool valid = r < nr;
    float part[MO];
#pragma unroll
    for (int j = 0; j < MO; ++j) part[j] = 0.f;
    for (int c = 2 * lane; c < 8 * ntl; c += 64) {
        const float* src = red + r * rs + c;
        float2 v = *reinterpret_cast<const float2*>(src);
#pragma unroll 4
        for (int q = 1; q < kg; ++q) {
            const float2 u = *reinterpret_cast<const float2*>(src + q * 16 * rs);
            v.x += u.x;
            v.y += u.y;
        }
        const float2 h = make_float2(fmaxf(v.x + bh[c], 0.f), fmaxf(v.y + bh[c + 1], 0.f));
        *reinterpret_cast<float2*>(hs + r * ld + c) = h;
        if (valid) *reinterpret_cast<float2*>(L.h_y + (long long)(r0 + r) * L.h_ldy + c) = h;
#pragma unroll
        for (int j = 0; j < MO; ++j)
            if (j < nout) part[j] = fmaf(h.x, wo[j * ldo + c], fmaf(h.y, wo[j * ldo + c + 1], part[j]));
    }
    float sv[MO], dv[MO];
    const float* bo = wo + ceil8(nout) * ldo;
#pragma unroll
    for (int j = 0; j < MO; ++j) {
        if (j < nout) {
            float t = part[j];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
            sv[j] = t + bo[j];
        }
    }
    const float li = loss_row(sv, nout, valid ? y[r] : 0, loss, inv_b, dv);
    if (!valid)
#pragma unroll
        for (int j = 0; j < MO; ++j) dv[j] = 0.f;
    if (valid && lane == 0) {
        rowloss[r] = li;
        float* lo = L.o_y + (long long)(r0 + r) * L.o_ldy;
        float* dl = L.o_d + (long long)(r0 + r) * L.o_ldd;
        for (int j = 0; j < nout; ++j) {
            lo[j] = sv[j];
            dl[j] = dv[j];
        }
    }
    __syncwarp();
    for (int c = 2 * lane; c < 8 * ntl; c += 64) {
        float g0 = 0.f, g1 = 0.f;
#pragma unroll
        for (int j = 0; j < MO; ++j)
            if (j < nout) {
                g0 = fmaf(dv[j], wo[j * ldo + c], g0);
                g1 = fmaf(dv[j], wo[j * ldo + c + 1], g1);
            }
        const float2 h = *reinterpret_cast<const float2*>(hs + r * ld + c);
        const float2 gd = make_float2(h.x > 0.f ? g0 : 0.f, h.y > 0.f ? g1 : 0.f);
        *reinterpret_cast<float2*>(gs + r * ld + c) = gd;
        if (valid) *reinterpret_cast<float2*>(L.h_d + (long long)(r0 + r) * L.h_ldd + c) = gd;
    }
}

__global__ void __launch_bounds__(NT, 1) fused_active_kernel(const FusedStepArgs a) {
    extern __shared__ __align__(16) float smem[];
    long long hdr_k = a.k;   // the embedding channel's header, read once the publisher has finished
    const int La = a.na, Lt = a.nt;
    const int ld = a.act_ld;
    float* ws = smem;
    // tiles of R x ld floats: 0 = x_a rows (later the logits); 1..La-1 = f_a's hidden
    // outputs; La = [z^a | z^p]; La+1..La+Lt-1 = g's hidden outputs; La+Lt, La+Lt+1 = gradients
    float* tiles = smem + a.w_floats;
    auto slot = [&](int i) { return tiles + i * R * ld; };
    float* X = slot(0);
    auto H = [&](int l) { return slot(1 + l); };            // output of f_a layer l < La - 1
    float* C = slot(La);
    auto TH = [&](int l) { return slot(La + 1 + l); };      // output of g layer l < Lt - 1
    float* G0 = slot(La + Lt);
    float* G1 = slot(La + Lt + 1);
    float* red = slot(La + Lt + 2);
    const FusedLayerArgs* A = a.L;
    const FusedLayerArgs* T = a.L + La;
    const int ea = A[La - 1].out;
    const int ep = T[0].in - ea;
    const int ep8 = ceil8(ep);
    const int nout = T[Lt - 1].out;
    const int ntiles = (a.rows + R - 1) / R;
    const float inv_b = 1.0f / (float)a.rows;
    const int Ltot = La + Lt;
    // one 16-row tile per CTA (the launch has one CTA per tile)
    if ((int)blockIdx.x >= ntiles) {
        griddep_wait();
        return;
    }
    {
        const int r0 = blockIdx.x * R;
        const int nr = min(R, a.rows - r0);
        async_rows(X, ld, a.x + (long long)r0 * a.ldx, a.ldx, (int)A[0].in_ld, nr);
        // one commit group per layer, in the order the forward uses them (group 0 also x^a's rows);
        // z^p's rows follow once the publisher has finished, after f_a's forward
        for (int l = 0; l < Ltot; ++l) {
            stage_layer_weights(ws, a.L[l]);
            cp_commit();
        }
        for (int l = 0; l < La; ++l) {                                   // z^a = f_a(x^a)
            cp_wait_pending(Ltot - 1 - l);       // x^a's rows and layers 0..l
            tile_fwd(l == 0 ? X : H(l - 1), ld, A[l].in, ws + A[l].ws_off, A[l].ws_ld, staged_bias(ws, A[l]), A[l].out,
                     A[l].fmap, l == La - 1 ? C : H(l), A[l].Y + (long long)r0 * A[l].ldy, A[l].ldy, nr, red);
        }
        griddep_wait();                                                  // the embedding's publisher has finished
        if (threadIdx.x == 0) hdr_k = a.chk_hdr->k;
        async_rows(C + ea, ld, a.zp + (long long)r0 * a.ldzp, a.ldzp, ep8, nr);   // beside z^a's columns
        cp_commit();
        // with n_out <= kFusedMaxOut, g's output layer, the loss, d(logits) and the output layer's input
        // gradient ride in the epilogue of g's last hidden layer (one warp per row)
        const bool fuse_out = Lt >= 2 && nout <= kFusedMaxOut;
        for (int l = 0; l < Lt - 1; ++l) {                               // g's hidden layers on [z^a | z^p]
            if (l == 0) {
                cp_wait_pending(0);                                      // z^p's rows (and every weight)
                const int r = threadIdx.x >> 5;                          // z^p kept for the update
                if (r < nr)
                    for (int c = threadIdx.x & 31; c < ep; c += 32)
                        a.zpc[(long long)(r0 + r) * a.ldzpc + c] = C[r * ld + ea + c];
            } else {
                __syncthreads();
            }
            if (fuse_out && l == Lt - 2) {
                const FusedLayerArgs& Lh = T[l];
                const FusedLayerArgs& Lo = T[Lt - 1];
                const TopLast tl{Lh.in, Lh.out, Lh.fmap, Lh.ws_off, Lh.ws_ld, Lo.out, Lo.ws_off, Lo.ws_ld,
                                 Lh.Y, Lh.ldy, Lh.D, Lh.ldd, Lo.Y, Lo.ldy, Lo.D, Lo.ldd};
                if (nout == 1)
                    top_last_fused<1>(l == 0 ? C : TH(l - 1), ld, ws, tl, TH(l), G0, a.y + r0, a.loss, inv_b,
                                      a.rowloss + r0, r0, nr, red);
                else
                    top_last_fused<kFusedMaxOut>(l == 0 ? C : TH(l - 1), ld, ws, tl, TH(l), G0, a.y + r0, a.loss,
                                                 inv_b, a.rowloss + r0, r0, nr, red);
            } else {
                tile_fwd(l == 0 ? C : TH(l - 1), ld, T[l].in, ws + T[l].ws_off, T[l].ws_ld, staged_bias(ws, T[l]),
                         T[l].out, T[l].fmap, TH(l), T[l].Y + (long long)r0 * T[l].ldy, T[l].ldy, nr, red);
            }
        }
        if (!fuse_out) {
            float* lg = X;                                               // x_a's tile is free again
            {                                                            // logits: no activation
                const FusedLayerArgs& L = T[Lt - 1];
                cp_wait_pending(0);
                if (Lt == 1) {                                           // z^p kept for the update
                    const int r = threadIdx.x >> 5;
                    if (r < nr)
                        for (int c = threadIdx.x & 31; c < ep; c += 32)
                            a.zpc[(long long)(r0 + r) * a.ldzpc + c] = C[r * ld + ea + c];
                }
                const float* bias = staged_bias(ws, L);
                float* yg = L.Y + (long long)r0 * L.ldy;
                const long long ldy = L.ldy;
                tile_gemm<false>(Lt == 1 ? C : TH(Lt - 2), ld, ceil8(L.in) / 8, ws + L.ws_off, L.ws_ld, ceil8(nout) / 8,
                                 L.fmap, red, [&](int r, int c, float v0, float v1) {
                                     v0 += bias[c];
                                     v1 += bias[c + 1];
                                     *reinterpret_cast<float2*>(lg + r * ld + c) = make_float2(v0, v1);
                                     if (r < nr) {
                                         if (c < nout) yg[(long long)r * ldy + c] = v0;
                                         if (c + 1 < nout) yg[(long long)r * ldy + c + 1] = v1;
                                     }
                                 });
            }
            __syncthreads();
            if (threadIdx.x < R) {                                       // loss, d(logits)
                const int r = threadIdx.x;
                const float* sr = lg + r * ld;
                float* d = G0 + r * ld;
                float* dg = T[Lt - 1].D + (long long)(r0 + r) * T[Lt - 1].ldd;
                if (r < nr) {
                    a.rowloss[r0 + r] = loss_row(sr, nout, a.y[r0 + r], a.loss, inv_b, d);
                    for (int j = 0; j < nout; ++j) dg[j] = d[j];
                } else {
                    for (int j = 0; j < nout; ++j) d[j] = 0.f;
                }
                for (int j = nout; j < ceil8(nout); ++j) d[j] = 0.f;
            }
        }
        griddep_trigger();   // the passive backward and the update may launch and stage now
        // backward through g: the input-gradient chain (from the last hidden layer when it was fused)
        float* gin = G0;
        float* gout = G1;
        for (int l = fuse_out ? Lt - 2 : Lt - 1; l >= 1; --l) {
            __syncthreads();
            tile_dx(gin, ld, T[l].out, ws + T[l].ws_off, T[l].ws_ld, T[l].in, T[l].dmap, TH(l - 1), gout,
                    T[l - 1].D + (long long)r0 * T[l - 1].ldd, T[l - 1].ldd, nr, red);
            float* t = gin;
            gin = gout;
            gout = t;
        }
        __syncthreads();
        {
            // g's first layer: [dz^a | dz^p] = dY W; dz^a * [z^a > 0] is the d(pre) of f_a's last
            // layer, dz^p (no mask: the passive party applies its own) is published
            const FusedLayerArgs& L = T[0];
            float* da = A[La - 1].D + (long long)r0 * A[La - 1].ldd;
            const long long ldda = A[La - 1].ldd;
            float* gp = a.gradp + (long long)r0 * a.ldgp;
            const long long ldgp = a.ldgp;
            float* go = gout;
            tile_gemm<true>(gin, ld, ceil8(L.out) / 8, ws + L.ws_off, L.ws_ld, ceil8(L.in) / 8, L.dmap, red,
                            [&](int r, int c, float v0, float v1) {
                                if (c < ea) {
                                    const float2 m = *reinterpret_cast<const float2*>(C + r * ld + c);
                                    const float2 v = make_float2(m.x > 0.f ? v0 : 0.f, m.y > 0.f ? v1 : 0.f);
                                    *reinterpret_cast<float2*>(go + r * ld + c) = v;
                                    if (r < nr) *reinterpret_cast<float2*>(da + (long long)r * ldda + c) = v;
                                } else if (r < nr) {
                                    *reinterpret_cast<float2*>(gp + (long long)r * ldgp + (c - ea)) = make_float2(v0, v1);
                                }
                            });
            float* t = gin;
            gin = gout;
            gout = t;
        }
        for (int l = La - 1; l >= 1; --l) {                              // backward through f_a
            __syncthreads();
            tile_dx(gin, ld, A[l].out, ws + A[l].ws_off, A[l].ws_ld, A[l].in, A[l].dmap, H(l - 1), gout,
                    A[l - 1].D + (long long)r0 * A[l - 1].ldd, A[l - 1].ldd, nr, red);
            float* t = gin;
            gin = gout;
            gout = t;
        }
    }
    if (threadIdx.x == 0 && hdr_k != a.k) atomicOr(a.status, ST_VERSION);
    publish_header(a.pub_hdr, a.k, a.batch, a.version);
}

__global__ void __launch_bounds__(NT, 1) fused_passive_bwd_kernel(const FusedStepArgs a) {
    extern __shared__ __align__(16) float smem[];
    griddep_trigger();       // the passive update may launch now (it waits for this grid before reading)
    long long hdr_k = a.k;   // the gradient channel's header, read once the active step has finished
    const int Lp = a.na;
    const int ld = a.act_ld;
    float* ws = smem;
    // tiles: 0..Lp-1 = f_p's outputs (saved by the forward), Lp = dz^p rows, Lp+1, Lp+2 = gradients
    float* tiles = smem + a.w_floats;
    auto slot = [&](int i) { return tiles + i * R * ld; };
    float* gs = slot(Lp);
    float* G0 = slot(Lp + 1);
    float* G1 = slot(Lp + 2);
    float* red = slot(Lp + 3);
    const FusedLayerArgs* P = a.L;
    const int ep8 = ceil8(P[Lp - 1].out);
    const int ntiles = (a.rows + R - 1) / R;
    // one 16-row tile per CTA (the launch has one CTA per tile)
    if ((int)blockIdx.x >= ntiles) {
        griddep_wait();
        return;
    }
    {
        const int r0 = blockIdx.x * R;
        const int nr = min(R, a.rows - r0);
        for (int l = 0; l < Lp; ++l)
            async_rows(slot(l), ld, P[l].Y + (long long)r0 * P[l].ldy, P[l].ldy, (int)P[l].out_ld, nr);
        cp_commit();
        // weights in the order the backward uses them (layer Lp-1 first), then wait for the active
        // step, whose dz^p comes last
        for (int l = Lp - 1; l >= 1; --l) {
            stage_layer_weights(ws, P[l]);
            cp_commit();
        }
        griddep_wait();
        if (threadIdx.x == 0) hdr_k = a.chk_hdr->k;
        async_rows(gs, ld, a.gradp + (long long)r0 * a.ldgp, a.ldgp, (int)P[Lp - 1].out_ld, nr);
        cp_commit();
        cp_wait_pending(0);
        {                                                                // dz^p * [z^p > 0]
            const int r = threadIdx.x >> 5;
            // DP on the embedding: the straight-through backward scales the received gradient by c
            const float sc = a.rowscale && r < nr ? a.rowscale[r0 + r] : 1.0f;
            const float* zp = slot(Lp - 1);
            float* dg = P[Lp - 1].D + (long long)(r0 + r) * P[Lp - 1].ldd;
            for (int c = (threadIdx.x & 31) * 2; c < ep8; c += 64) {
                const float2 z = *reinterpret_cast<const float2*>(zp + r * ld + c);
                const float2 gr = *reinterpret_cast<const float2*>(gs + r * ld + c);
                const float2 v = make_float2(z.x > 0.f ? sc * gr.x : 0.f, z.y > 0.f ? sc * gr.y : 0.f);
                *reinterpret_cast<float2*>(G0 + r * ld + c) = v;
                if (r < nr) *reinterpret_cast<float2*>(dg + c) = v;
            }
        }
        float* gin = G0;
        float* gout = G1;
        for (int l = Lp - 1; l >= 1; --l) {
            __syncthreads();
            tile_dx(gin, ld, P[l].out, ws + P[l].ws_off, P[l].ws_ld, P[l].in, P[l].dmap, slot(l - 1), gout,
                    P[l - 1].D + (long long)r0 * P[l - 1].ldd, P[l - 1].ldd, nr, red);
            float* t = gin;
            gin = gout;
            gout = t;
        }
    }
    if (threadIdx.x == 0 && hdr_k != a.k) atomicOr(a.status, ST_VERSION);
}

// dW = D^T X, db = sum of D's rows, then SGD, for one 32 x 32 output tile per
// cluster; CTA `rank` of the cluster covers rows [rank c, (rank + 1) c) with
// c = ceil(rows / 8).  Inside a CTA, 4 row groups accumulate in fp32 and are
// summed in a fixed order; each CTA then pushes its partial of the 128 outputs
// rank q owns into q's shared memory (slot = sender's rank), and after one
// cluster barrier every owner sums its 8 slots in rank order and applies SGD.
constexpr int kUpdRows = 128;                // rows staged per pass: 32 per row group of 2 warps
constexpr int kUpdLd = kUpdTile + 8;         // smem row stride, 8 mod 32: the MMA fragment loads are conflict-free
static_assert(kUpdThreads == 256 && kUpdTile == 32, "the thread map below assumes 256 threads and 32 x 32 tiles");
static_assert(kUpdThreads == 256 && kUpdRows == 128, "4 row groups x 2 warps, 32 rows per group");
static_assert(2 * kUpdRows * kUpdLd >= 4 * kUpdTile * kUpdTile, "the row-group partials reuse the stage");

__global__ void __cluster_dims__(kUpdCluster, 1, 1) __launch_bounds__(kUpdThreads)
    fused_update_kernel(const FusedUpdArgs a) {
    __shared__ __align__(16) float stage[2 * kUpdRows * kUpdLd];
    float* Ds = stage;
    float* Xs = stage + kUpdRows * kUpdLd;
    constexpr int kPer = kUpdTile * kUpdTile / kUpdCluster;   // outputs of the tile each rank owns
    constexpr int kPerB = kUpdTile / kUpdCluster;             // bias outputs each rank owns
    __shared__ __align__(16) float Rw[kUpdCluster * kPer];    // partials of the owned outputs, by sender
    __shared__ float Rb[kUpdCluster * kPerB];
    __shared__ float Pb[kUpdThreads / 32];                    // the loss cluster's warp sums
    // a passive forward that reads the version this update writes may launch now and fetch its rows; it
    // waits for this grid before it reads the weights
    griddep_trigger();
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int tile = blockIdx.x / kUpdCluster;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // the d(pre-activation) rows, most inputs X and the row losses come from the row kernel this launch
    // depends on (programmatically, in a graph): griddep_wait() comes before any read of them
    if (tile == a.ntiles) {                                  // one extra cluster: mean loss of the step, fixed order
        griddep_wait();
        if (rank == 0 && a.loss_out) {
            float s = 0.f;
            for (int r = tid; r < a.rows; r += kUpdThreads) s += a.rowloss[r];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) s += __shfl_down_sync(0xffffffffu, s, o);
            if (lane == 0) Pb[warp] = s;
            __syncthreads();
            if (tid == 0) {
                float v = 0.f;
                for (int w = 0; w < kUpdThreads / 32; ++w) v += Pb[w];
                *a.loss_out = v / (float)a.rows;
                if (a.loss_host) *a.loss_host = v / (float)a.rows;
            }
        }
        return;
    }
    int l = 0;
    while (l + 1 < a.nl && tile >= a.L[l + 1].tile0) ++l;
    const FusedUpdLayer& L = a.L[l];
    const int t = tile - L.tile0;
    const int o0 = (t / L.tiles_i) * kUpdTile, i0 = (t % L.tiles_i) * kUpdTile;
    const int no = min(kUpdTile, L.out - o0), ni = min(kUpdTile, L.in - i0);
    const bool bias = i0 == 0;
    const int chunk = (a.rows + kUpdCluster - 1) / kUpdCluster;
    const int rbeg = min(a.rows, rank * chunk), rend = min(a.rows, rbeg + chunk);
    // this rank's outputs of the tile: the master of version k was written by the previous update, a
    // full dependency, so it is read now and its latency hides behind the wait
    const int eo = rank * kPer + tid, oo = eo / kUpdTile, io = eo - oo * kUpdTile;
    const bool own_w = tid < kPer && oo < no && io < ni;
    const long long widx = (long long)(o0 + oo) * L.in + (i0 + io);
    const float wm = own_w ? L.Wm[widx] : 0.f;
    const int ob = rank * kPerB + (tid - kPer);
    const bool own_b = bias && tid >= kPer && tid < kPer + kPerB && ob < no;
    const float bmv = own_b ? L.bm[o0 + ob] : 0.f;
    // rows [rb, rb + nr) of X[:, i0 : i0+32] in 16-byte chunks (cp.async), zero past the layer's columns;
    // X's columns come from X or, from xsplit on (a multiple of 4), from X2
    auto stage_x = [&](int rb, int nr) {
        for (int e = tid; e < kUpdRows * (kUpdTile / 4); e += kUpdThreads) {
            const int r = e >> 3, c = (e & 7) * 4;
            float* xs = Xs + r * kUpdLd + c;
            const long long gr = rb + r;
            const int ic = i0 + c;
            if (r < nr && ic < L.in)
                cp16(xs, ic < L.xsplit ? L.X + gr * L.ldx + ic : L.X2 + gr * L.ldx2 + (ic - L.xsplit));
            else
                *reinterpret_cast<float4*>(xs) = make_float4(0.f, 0.f, 0.f, 0.f);
        }
    };
    if (L.x_early && rbeg < rend) stage_x(rbeg, min(kUpdRows, rend - rbeg));
    griddep_wait();

    const int fg = lane >> 2, ft = lane & 3;     // MMA fragment row / column lane
    // the 32 x 32 tile as 2 (outputs) x 4 (inputs) MMA blocks in 3xTF32, A[o][r] = D[r][o],
    // B[r][i] = X[r][i]: warp w takes output half mt = w mod 2 and the 32 rows of row group w / 2
    const int mt = warp & 1, rgrp = warp >> 1;
    float acc[4][4];
#pragma unroll
    for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[nt][q] = 0.f;
    float bacc = 0.f;                                        // db partial of output tid & 31
    const bool dvec = (L.ldd & 3) == 0;                      // D rows hold whole 16-byte chunks
    for (int rb = rbeg; rb < rend; rb += kUpdRows) {
        const int nr = min(kUpdRows, rend - rb);
        if (rb > rbeg) __syncthreads();                      // the previous pass has read the stage
        // rows [rb, rb + nr) of D[:, o0 : o0+32] in 16-byte chunks (cp.async), zero past the layer's columns
        for (int e = tid; e < kUpdRows * (kUpdTile / 4); e += kUpdThreads) {
            const int r = e >> 3, c = (e & 7) * 4;
            float* ds = Ds + r * kUpdLd + c;
            const long long gr = rb + r;
            if (r < nr && o0 + c < L.out && dvec) {
                cp16(ds, L.D + gr * L.ldd + o0 + c);
            } else {
#pragma unroll
                for (int q = 0; q < 4; ++q) ds[q] = (r < nr && o0 + c + q < L.out) ? __ldg(L.D + gr * L.ldd + o0 + c + q) : 0.f;
            }
        }
        if (!(L.x_early && rb == rbeg)) stage_x(rb, nr);
        cp_commit();
        cp_wait_pending(0);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            const int k0 = rgrp * 32 + kk * 8;               // rows past nr are zero-filled
            uint32_t ah[4], al[4], bh[4][2], bl[4][2];
            const float* d0 = Ds + (k0 + ft) * kUpdLd + mt * 16 + fg;
            const float* d1 = d0 + 4 * kUpdLd;
            split_tf32(d0[0], ah[0], al[0]);
            split_tf32(d0[8], ah[1], al[1]);
            split_tf32(d1[0], ah[2], al[2]);
            split_tf32(d1[8], ah[3], al[3]);
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
                const float* x0 = Xs + (k0 + ft) * kUpdLd + nt * 8 + fg;
                split_tf32(x0[0], bh[nt][0], bl[nt][0]);
                split_tf32(x0[4 * kUpdLd], bh[nt][1], bl[nt][1]);
            }
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) mma_tf32(acc[nt], al, bh[nt]);
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) mma_tf32(acc[nt], ah, bl[nt]);
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) mma_tf32(acc[nt], ah, bh[nt]);
        }
        if (bias)
            for (int r = tid >> 5; r < nr; r += kUpdThreads / 32) bacc += Ds[r * kUpdLd + (tid & 31)];
    }
    __shared__ float bpart[kUpdThreads];                     // db partials [8 warps][32]
    bpart[tid] = bacc;
    __syncthreads();
    float* gpart = stage;                                    // [4 row groups][32][32]
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
        float* pw = gpart + rgrp * kUpdTile * kUpdTile + (mt * 16 + fg) * kUpdTile + nt * 8 + 2 * ft;
        *reinterpret_cast<float2*>(pw) = make_float2(acc[nt][0], acc[nt][1]);
        *reinterpret_cast<float2*>(pw + 8 * kUpdTile) = make_float2(acc[nt][2], acc[nt][3]);
    }
    __syncthreads();
    // rank q owns outputs [128 q, 128 q + 128) of the tile (rows 4q..4q+3) and bias outputs 4q..4q+3
    for (int e = tid; e < kUpdTile * kUpdTile; e += kUpdThreads) {
        const float v = ((gpart[e] + gpart[1024 + e]) + gpart[2048 + e]) + gpart[3072 + e];
        const int q = e / kPer;
        cluster.map_shared_rank(Rw, q)[rank * kPer + (e - q * kPer)] = v;
    }
    if (tid < kUpdTile) {
        float sb = 0.f;
        for (int w = 0; w < kUpdThreads / 32; ++w) sb += bpart[w * 32 + tid];
        const int q = tid / kPerB;
        cluster.map_shared_rank(Rb, q)[rank * kPerB + (tid - q * kPerB)] = sb;
    }
    cluster.sync();   // every push has landed; no shared memory of another CTA is touched after this
    if (own_w) {
        float g = 0.f;
#pragma unroll
        for (int q = 0; q < kUpdCluster; ++q) g += Rw[q * kPer + tid];
        L.gW[widx] = g;
        const float w = wm - a.lr * g;
        L.Wm[widx] = w;
        L.Wc[(long long)(o0 + oo) * L.in_ld + (i0 + io)] = w;
    } else if (own_b) {
        float g = 0.f;
#pragma unroll
        for (int q = 0; q < kUpdCluster; ++q) g += Rb[q * kPerB + (tid - kPer)];
        const int go = o0 + ob;
        L.gb[go] = g;
        const float b = bmv - a.lr * g;
        L.bm[go] = b;
        L.bc[go] = b;
    }
}

template <typename K>
cudaError_t set_smem_attr(K kernel) {
    // every fused kernel asks for the largest shared-memory carveout, so an SM
    // moving from one of them to the next keeps its L1 / shared split
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFusedMaxSmem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    return e;
}

// Launch with the programmatic-launch attributes of `o` (a plain launch when it asks for none).
template <typename Args>
cudaError_t launch_with(void (*kernel)(const Args), const Args& a, int grid, int block, size_t smem, cudaStream_t s,
                        const LaunchOpt& o) {
    if (!o.serialize && !o.pevent) {
        kernel<<<grid, block, smem, s>>>(a);
        return cudaGetLastError();
    }
    cudaLaunchAttribute at[2];
    int n = 0;
    if (o.serialize) {
        at[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        at[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    if (o.pevent) {
        at[n].id = cudaLaunchAttributeProgrammaticEvent;
        at[n].val.programmaticEvent.event = o.pevent;
        at[n].val.programmaticEvent.flags = 0;
        at[n].val.programmaticEvent.triggerAtBlockStart = 0;
        ++n;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = at;
    cfg.numAttrs = n;
    return cudaLaunchKernelEx(&cfg, kernel, a);
}

}  // namespace

cudaError_t launch_fused_passive_fwd(const FusedChainArgs& a, cudaStream_t s, const LaunchOpt& o) {
    static cudaError_t attr = set_smem_attr(fused_passive_fwd_kernel);
    if (attr != cudaSuccess) return attr;
    const int ntiles = (a.rows + R - 1) / R;
    return launch_with(fused_passive_fwd_kernel, a, ntiles, NT, fused_smem_fwd(a.w_floats, a.act_ld), s, o);
}

cudaError_t launch_fused_active(const FusedStepArgs& a, cudaStream_t s, const LaunchOpt& o) {
    static cudaError_t attr = set_smem_attr(fused_active_kernel);
    if (attr != cudaSuccess) return attr;
    const int ntiles = (a.rows + R - 1) / R;
    return launch_with(fused_active_kernel, a, ntiles, NT, fused_smem_active(a.w_floats, a.act_ld, a.na, a.nt), s, o);
}

cudaError_t launch_fused_passive_bwd(const FusedStepArgs& a, cudaStream_t s, const LaunchOpt& o) {
    static cudaError_t attr = set_smem_attr(fused_passive_bwd_kernel);
    if (attr != cudaSuccess) return attr;
    const int ntiles = (a.rows + R - 1) / R;
    return launch_with(fused_passive_bwd_kernel, a, ntiles, NT, fused_smem_pbwd(a.w_floats, a.act_ld, a.na), s, o);
}

cudaError_t launch_fused_update(const FusedUpdArgs& a, cudaStream_t s, const LaunchOpt& o) {
    static cudaError_t attr = cudaFuncSetAttribute(fused_update_kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (attr != cudaSuccess) return attr;
    if (a.ntiles < 1 || a.rows < 1) return cudaErrorInvalidValue;
    // one more cluster than output tiles when the step's mean loss is wanted
    return launch_with(fused_update_kernel, a, (a.ntiles + (a.loss_out ? 1 : 0)) * kUpdCluster, kUpdThreads, 0, s, o);
}

bool is_fused_kernel(const void* func) {
    return func == reinterpret_cast<const void*>(fused_passive_fwd_kernel) ||
           func == reinterpret_cast<const void*>(fused_active_kernel) ||
           func == reinterpret_cast<const void*>(fused_passive_bwd_kernel) ||
           func == reinterpret_cast<const void*>(fused_update_kernel);
}

}  // namespace vfl
