// Fused kernels for narrow fp32 models (every width <= 256, one worker stream
// per party): each phase of Algorithm 1 is one launch.
//
//  - passive forward: every CTA stages all of f_p's weights (transposed copies)
//    into shared memory with cp.async, then runs the bottom chain for its row
//    tile; the last CTA to finish publishes the channel header.
//  - active step (cooperative launch): phase 1 is row-parallel -- active bottom
//    forward, top forward on [z^a | z^p], loss, the input-gradient chain back to
//    the first active layer, publish dz^p, and each row tile's partial weight
//    gradient (from the tiles already in shared memory).  After a grid-wide
//    barrier, phase 2 sums the partials of every parameter over the row tiles
//    in a fixed order (deterministic) and applies SGD to the master and the new
//    version's copies; CTA 0 reduces the loss and writes the gradient header.
//  - passive backward (cooperative launch): the same two phases for f_p.
#include <cooperative_groups.h>

#include "vfl_fused.cuh"

namespace cg = cooperative_groups;

namespace vfl {

namespace {

constexpr int NT = kFusedThreads;     // 16 warps
constexpr int R = kFusedRows;
static_assert(R == 16, "the MMA tiles cover exactly 16 rows");

__device__ __forceinline__ void cp16(float* s, const float* g) {
    const unsigned sa = (unsigned)__cvta_generic_to_shared(s);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(sa), "l"(g) : "memory");
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
__device__ void async_rows(float* s, int lds, const float* g, long long ldg, int cols, int nrows) {
    const int q = cols / 4;
    for (int i = threadIdx.x; i < R * q; i += NT) {
        const int r = i / q, c = (i - r * q) * 4;
        if (r < nrows)
            cp16(s + r * lds + c, g + (long long)r * ldg + c);
        else
            *reinterpret_cast<float4*>(s + r * lds + c) = make_float4(0.f, 0.f, 0.f, 0.f);
    }
}

// rows x cols floats (cols % 4 == 0, 16-byte aligned rows) into smem rows of stride lds, asynchronously
__device__ void async_matrix(float* s, int lds, const float* g, long long ldg, int rows, int cols) {
    const int q = cols / 4;
    for (int i = threadIdx.x; i < rows * q; i += NT) {
        const int r = i / q, c = (i - r * q) * 4;
        cp16(s + r * lds + c, g + (long long)r * ldg + c);
    }
}

__device__ void stage_layer_weights(float* ws, const FusedLayerArgs& L) {
    if (L.ws_off >= 0) async_matrix(ws + L.ws_off, L.ws_ld, L.W, L.in_ld, L.out, (int)L.in_ld);
}

// ---- warp-level tensor-core tiles: mma.sync m16n8k8 TF32 in 3xTF32 form ----
// Each fp32 operand x is split into hi = tf32(x) and lo = tf32(x - hi); the
// product is accumulated as lo*hi + hi*lo + hi*hi in fp32 (the lo*lo term,
// ~2^-22 relative, is dropped), which keeps fp32-level accuracy.
__device__ __forceinline__ uint32_t to_tf32(float x) {
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return r;
}

__device__ __forceinline__ void split_tf32(float x, uint32_t& hi, uint32_t& lo) {
    hi = to_tf32(x);
    lo = to_tf32(x - __uint_as_float(hi));
}

__device__ __forceinline__ void mma_tf32(float* d, const uint32_t* a, const uint32_t* b) {
    asm volatile(
        "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// d += a_hi*b_hi and e += a_lo*b_hi + a_hi*b_lo for a 16x8 (A) by 8x8 (B)
// fragment pair given as fp32 values; the caller adds e into d at the end
// (two accumulators keep the dependent MMA chain short).
__device__ __forceinline__ void mma_3xtf32(float* d, float* e, const float* a, const float* b) {
    uint32_t ah[4], al[4], bh[2], bl[2];
#pragma unroll
    for (int i = 0; i < 4; ++i) split_tf32(a[i], ah[i], al[i]);
    split_tf32(b[0], bh[0], bl[0]);
    split_tf32(b[1], bh[1], bl[1]);
    mma_tf32(e, al, bh);
    mma_tf32(d, ah, bh);
    mma_tf32(e, ah, bl);
}

// One 16x8 output tile of  sum_k A[r][k] B[k][n]  for k in [kbeg, kend), 3xTF32.
// A is the 16-row tile (row stride lda, columns past K masked); B[k][n] is read
// as  bm[n * ldb_n + k * ldb_k]  (rows past N / K masked).  Accumulates into d, e.
__device__ __forceinline__ void mma_tile_range(float* d, float* e, const float* as, int lda, int K, const float* bm,
                                               int ldb_n, int ldb_k, int n, bool n_ok, int kbeg, int kend) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    for (int k0 = kbeg; k0 < kend; k0 += 8) {
        const int ka = k0 + t, kb = k0 + t + 4;
        float a[4], b[2];
        a[0] = ka < K ? as[g * lda + ka] : 0.f;
        a[1] = ka < K ? as[(g + 8) * lda + ka] : 0.f;
        a[2] = kb < K ? as[g * lda + kb] : 0.f;
        a[3] = kb < K ? as[(g + 8) * lda + kb] : 0.f;
        b[0] = (ka < K && n_ok) ? bm[n * ldb_n + ka * ldb_k] : 0.f;
        b[1] = (kb < K && n_ok) ? bm[n * ldb_n + kb * ldb_k] : 0.f;
        mma_3xtf32(d, e, a, b);
    }
}

// C[16 x N] = A[16 x K] . B over the 16 warps of the block: output tile j (8
// columns) goes to warp j mod 16; with at most 8 tiles the K range is split
// between warps w and w + 8 and the second half is added through `red`
// (fixed order).  The epilogue callback receives (row, col, value) for
// every in-range output.
template <typename Epi>
__device__ void tile_gemm(const float* as, int lda, int K, const float* bm, int ldb_n, int ldb_k, int N, float* red,
                          Epi epi) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, g = lane >> 2, t = lane & 3;
    constexpr int NW = NT / 32;
    const int ntiles = (N + 7) / 8;
    const bool split = ntiles <= NW / 2;
    const int ksteps = (K + 7) / 8;
    const int khalf = ((ksteps + 1) / 2) * 8;
    float d[2][4] = {}, e[2][4] = {};
    int mine = 0;
    if (split) {
        const int j = warp % (NW / 2), half = warp / (NW / 2);
        if (j < ntiles) {
            const int n = j * 8 + g;
            mma_tile_range(d[0], e[0], as, lda, K, bm, ldb_n, ldb_k, n, n < N, half ? khalf : 0, half ? K : min(K, khalf));
            mine = 1;
        }
        if (mine && half) {
#pragma unroll
            for (int q = 0; q < 4; ++q) red[(j * 32 + lane) * 4 + q] = d[0][q] + e[0][q];
        }
        __syncthreads();
        if (!mine || half) return;
#pragma unroll
        for (int q = 0; q < 4; ++q) d[0][q] += e[0][q] + red[(j * 32 + lane) * 4 + q];
        const int c0 = j * 8 + 2 * t;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int c = c0 + (q & 1);
            if (c < N) epi(g + 8 * (q >> 1), c, d[0][q]);
        }
        return;
    }
#pragma unroll
    for (int jj = 0; jj < 2; ++jj) {
        const int j = warp + NW * jj;
        if (j < ntiles) {
            const int n = j * 8 + g;
            mma_tile_range(d[jj], e[jj], as, lda, K, bm, ldb_n, ldb_k, n, n < N, 0, K);
        }
    }
#pragma unroll
    for (int jj = 0; jj < 2; ++jj) {
        const int j = warp + NW * jj;
        if (j >= ntiles) break;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int c = j * 8 + 2 * t + (q & 1);
            if (c < N) epi(g + 8 * (q >> 1), c, d[jj][q] + e[jj][q]);
        }
    }
}

// Y[r][c] = act(sum_k X[r][k] W[c][k] + b[c]) for the 16 rows of a tile (W
// row-major in smem).  To smem (ldy) and to global rows < nrows when yg is set.
__device__ void tile_fwd(const float* xs, int ldx, int K, const float* ws, int ldw, const float* __restrict__ bias,
                         int N, bool relu, float* ys, int ldy, float* yg, long long ldyg, int nrows, float* red) {
    tile_gemm(xs, ldx, K, ws, ldw, 1, N, red, [&](int r, int c, float v) {
        float y = v + bias[c];
        if (relu) y = fmaxf(y, 0.f);
        ys[r * ldy + c] = y;
        if (yg && r < nrows) yg[(long long)r * ldyg + c] = y;
    });
}

// dX[r][k] = sum_c dY[r][c] W[c][k], zeroed where prev[r][k] <= 0 (when prev is
// given).  To smem and to global rows < nrows.
__device__ void tile_dx(const float* dys, int ldd, int N, const float* ws, int ldw, int K, const float* prev, int ldp,
                        float* os, int ldo, float* og, long long ldog, int nrows, float* red) {
    tile_gemm(dys, ldd, N, ws, 1, ldw, K, red, [&](int r, int k, float v) {
        if (prev && !(prev[r * ldp + k] > 0.f)) v = 0.f;
        os[r * ldo + k] = v;
        if (og && r < nrows) og[(long long)r * ldog + k] = v;
    });
}

// Partial gradient of one layer over the tile's 16 rows, [W | b] flat:
// part[o*in + k] = sum_r D[r][o] X[r][k] (16-output x 8-input MMA tiles, K = 16
// rows in two steps) and part[out*in + o] = sum_r D[r][o].  Rows beyond the
// batch hold D = 0; smem columns past out / in are masked.
__device__ void tile_partial(const float* Ds, int ldd, const float* Xs, int ldx, int out, int in,
                             float* __restrict__ part) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, g = lane >> 2, t = lane & 3;
    const int mt = (out + 15) / 16, nt = (in + 7) / 8;
    for (int it = warp; it < mt * nt; it += NT / 32) {
        const int o0 = (it / nt) * 16, i0 = (it % nt) * 8;
        const int oa = o0 + g, ob = o0 + g + 8, i = i0 + g;
        float d[4] = {0.f, 0.f, 0.f, 0.f}, e[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int r0 = 0; r0 < R; r0 += 8) {
            const float* d0 = Ds + (r0 + t) * ldd;
            const float* d1 = Ds + (r0 + t + 4) * ldd;
            float a[4], b[2];
            a[0] = oa < out ? d0[oa] : 0.f;
            a[1] = ob < out ? d0[ob] : 0.f;
            a[2] = oa < out ? d1[oa] : 0.f;
            a[3] = ob < out ? d1[ob] : 0.f;
            b[0] = i < in ? Xs[(r0 + t) * ldx + i] : 0.f;
            b[1] = i < in ? Xs[(r0 + t + 4) * ldx + i] : 0.f;
            mma_3xtf32(d, e, a, b);
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int o = o0 + g + 8 * (q >> 1), k = i0 + 2 * t + (q & 1);
            if (o < out && k < in) part[(long long)o * in + k] = d[q] + e[q];
        }
    }
    for (int o = threadIdx.x; o < out; o += NT) {
        float acc = 0.f;
#pragma unroll
        for (int r = 0; r < R; ++r) acc += Ds[r * ldd + o];
        part[(long long)out * in + o] = acc;
    }
}

// Phase 2: every parameter's gradient = sum of the row tiles' partials in tile
// order, then SGD (Eq. 2) on the master and on both copies of the new version.
__device__ void reduce_and_sgd(const FusedStepArgs& a, int nl, int ntiles) {
    for (long long i = blockIdx.x * (long long)NT + threadIdx.x; i < a.ptotal; i += (long long)gridDim.x * NT) {
        int l = 0;
        while (l + 1 < nl && i >= a.L[l + 1].poff) ++l;
        const FusedLayerArgs& L = a.L[l];
        float g = 0.f;
#pragma unroll 16
        for (int t = 0; t < ntiles; ++t) g += __ldcg(a.part + (long long)t * a.ptotal + i);
        const long long idx = i - L.poff;
        const long long nw = (long long)L.out * L.in;
        if (idx < nw) {
            L.gW[idx] = g;
            const float w = L.Wm[idx] - a.lr * g;
            L.Wm[idx] = w;
            const long long o = idx / L.in, k = idx - o * L.in;
            L.Wc[o * L.in_ld + k] = w;
        } else {
            const long long o = idx - nw;
            L.gb[o] = g;
            const float b = L.bm[o] - a.lr * g;
            L.bm[o] = b;
            L.bc[o] = b;
        }
    }
}

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(NT, 1) fused_passive_fwd_kernel(const FusedChainArgs a) {
    extern __shared__ __align__(16) float smem[];
    float* ws = smem;
    float* buf0 = smem + a.w_floats;
    float* buf1 = buf0 + R * a.act_ld;
    float* red = buf1 + R * a.act_ld;           // K-split partial sums of tile_gemm
    const int ntiles = (a.rows + R - 1) / R;
    bool first = true;
    for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int r0 = tile * R;
        const int nr = min(R, a.rows - r0);
        __syncthreads();
        async_rows(buf0, a.act_ld, a.x + (long long)r0 * a.ldx, a.ldx, (int)a.L[0].in_ld, nr);
        if (first) {
            // group l holds layer l's weights (group 0 also the first tile), so layer l only
            // waits for its own weights while the later ones are still arriving
            for (int l = 0; l < a.nl; ++l) {
                stage_layer_weights(ws, a.L[l]);
                cp_commit();
            }
        } else {
            cp_commit();
        }
        float* cur = buf0;
        float* nxt = buf1;
        for (int l = 0; l < a.nl; ++l) {
            const FusedLayerArgs& L = a.L[l];
            if (first)
                cp_wait_pending(a.nl - 1 - l);
            else if (l == 0)
                cp_wait_pending(0);
            else
                __syncthreads();
            tile_fwd(cur, a.act_ld, L.in, ws + L.ws_off, L.ws_ld, L.b, L.out, true, nxt, a.act_ld,
                     L.Y + (long long)r0 * L.ldy, L.ldy, nr, red);
            float* t = cur;
            cur = nxt;
            nxt = t;
        }
        first = false;
    }
    // the last CTA to finish publishes the header after every payload write
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const int done = atomicAdd(a.counter, 1);
        if (done == (int)gridDim.x - 1) {
            __threadfence();
            a.hdr->k = a.k;
            a.hdr->batch = a.batch;
            a.hdr->version = a.version;
            *a.counter = 0;
            __threadfence();
        }
    }
}

__global__ void __launch_bounds__(NT, 1) fused_active_kernel(const FusedStepArgs a) {
    extern __shared__ __align__(16) float smem[];
    cg::grid_group grid = cg::this_grid();
    const int La = a.na, Lt = a.nt;
    const int ldA = a.act_ld;
    float* ws = smem;
    float* acts = smem + a.w_floats;
    // slots: 0 = x_a; 1..La = f_a outputs; La+1 = [z^a | z^p]; La+2..La+1+Lt = g outputs (last: logits);
    // La+Lt+2, La+Lt+3 = gradient ping-pong
    auto act = [&](int i) { return acts + i * R * ldA; };
    float* g0 = act(La + Lt + 2);
    float* g1 = act(La + Lt + 3);
    float* red = act(La + Lt + 4);              // K-split partial sums of tile_gemm
    if (threadIdx.x == 0 && a.chk_hdr->k != a.k) atomicOr(a.status, ST_VERSION);
    const FusedLayerArgs* A = a.L;
    const FusedLayerArgs* T = a.L + La;
    const int ea = A[La - 1].out;
    const int ep = T[0].in - ea;
    const int nout = T[Lt - 1].out;
    const int ntiles = (a.rows + R - 1) / R;
    const float inv_b = 1.0f / (float)a.rows;
    bool first = true;
    for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int r0 = tile * R;
        const int nr = min(R, a.rows - r0);
        float* part = a.part + (long long)tile * a.ptotal;
        __syncthreads();
        async_rows(act(0), ldA, a.x + (long long)r0 * a.ldx, a.ldx, (int)A[0].in_ld, nr);
        async_rows(act(La + 1) + ea, ldA, a.zp + (long long)r0 * a.ldzp, a.ldzp, ep, nr);
        if (first) {
            // one commit group per layer, in the order the forward uses them
            for (int l = 0; l < La + Lt; ++l) {
                stage_layer_weights(ws, a.L[l]);
                cp_commit();
            }
        } else {
            cp_commit();
        }
        for (int l = 0; l < La; ++l) {                                   // z^a = f_a(x^a)
            if (first)
                cp_wait_pending(La + Lt - 1 - l);
            else if (l == 0)
                cp_wait_pending(0);
            else
                __syncthreads();
            tile_fwd(act(l), ldA, A[l].in, ws + A[l].ws_off, A[l].ws_ld, A[l].b, A[l].out, true, act(l + 1), ldA,
                     A[l].Y + (long long)r0 * A[l].ldy, A[l].ldy, nr, red);
        }
        __syncthreads();
        for (int i = threadIdx.x; i < R * ea; i += NT) {                 // [z^a | z^p]
            const int r = i / ea, c = i - r * ea;
            act(La + 1)[r * ldA + c] = act(La)[r * ldA + c];
        }
        for (int l = 0; l < Lt; ++l) {                                   // y_hat = g(z^a, z^p)
            if (first)
                cp_wait_pending(Lt - 1 - l);
            else
                __syncthreads();
            tile_fwd(act(La + 1 + l), ldA, T[l].in, ws + T[l].ws_off, T[l].ws_ld, T[l].b, T[l].out, l < Lt - 1,
                     act(La + 2 + l), ldA, T[l].Y + (long long)r0 * T[l].ldy, T[l].ldy, nr, red);
        }
        __syncthreads();
        if (threadIdx.x < R) {                                           // loss, d(logits)
            const int r = threadIdx.x;
            const float* s = act(La + 1 + Lt) + r * ldA;
            float* d = g0 + r * ldA;
            if (r < nr) {
                const int y = a.y[r0 + r];
                float li;
                if (a.loss == VFL_LOSS_BCE) {
                    const float x = s[0];
                    li = fmaxf(x, 0.f) - x * (float)y + log1pf(expf(-fabsf(x)));
                    d[0] = (1.0f / (1.0f + expf(-x)) - (float)y) * inv_b;
                } else {
                    float m = s[0];
                    for (int j = 1; j < nout; ++j) m = fmaxf(m, s[j]);
                    float z = 0.f;
                    for (int j = 0; j < nout; ++j) z += expf(s[j] - m);
                    li = logf(z) + m - s[y];
                    const float iz = 1.0f / z;
                    for (int j = 0; j < nout; ++j) d[j] = (expf(s[j] - m) * iz - (j == y ? 1.f : 0.f)) * inv_b;
                }
                a.rowloss[r0 + r] = li;
                for (int j = 0; j < nout; ++j) a.ds[(long long)(r0 + r) * nout + j] = d[j];
            } else {
                for (int j = 0; j < nout; ++j) d[j] = 0.f;
            }
        }
        // backward through g: partial gradients, input-gradient chain
        float* gin = g0;
        float* gout = g1;
        for (int l = Lt - 1; l >= 0; --l) {
            __syncthreads();
            tile_partial(gin, ldA, act(La + 1 + l), ldA, T[l].out, T[l].in, part + T[l].poff);
            if (l > 0)
                tile_dx(gin, ldA, T[l].out, ws + T[l].ws_off, T[l].ws_ld, T[l].in, act(La + 1 + l), ldA, gout, ldA,
                        T[l - 1].D + (long long)r0 * T[l - 1].ldd, T[l - 1].ldd, nr, red);
            else
                tile_dx(gin, ldA, T[l].out, ws + T[l].ws_off, T[l].ws_ld, T[l].in, nullptr, 0, gout, ldA, nullptr, 0,
                        nr, red);
            float* t = gin;
            gin = gout;
            gout = t;
        }
        __syncthreads();
        // split [dz^a | dz^p]: dz^a * [z^a > 0] is the d(pre) of f_a's last layer; dz^p is published
        for (int i = threadIdx.x; i < R * (ea + ep); i += NT) {
            const int r = i / (ea + ep), c = i - r * (ea + ep);
            float v = gin[r * ldA + c];
            if (c < ea) {
                if (!(act(La)[r * ldA + c] > 0.f)) v = 0.f;
                gout[r * ldA + c] = v;
                if (r < nr) A[La - 1].D[(long long)(r0 + r) * A[La - 1].ldd + c] = v;
            } else if (r < nr) {
                a.gradp[(long long)(r0 + r) * a.ldgp + (c - ea)] = v;
            }
        }
        gin = gout;
        gout = (gin == g0) ? g1 : g0;
        for (int l = La - 1; l >= 0; --l) {                              // backward through f_a
            __syncthreads();
            tile_partial(gin, ldA, act(l), ldA, A[l].out, A[l].in, part + A[l].poff);
            if (l > 0) {
                tile_dx(gin, ldA, A[l].out, ws + A[l].ws_off, A[l].ws_ld, A[l].in, act(l), ldA, gout, ldA,
                        A[l - 1].D + (long long)r0 * A[l - 1].ldd, A[l - 1].ldd, nr, red);
                float* t = gin;
                gin = gout;
                gout = t;
            }
        }
        first = false;
    }
    if (first) cp_wait_pending(0);   // CTAs without a row tile have nothing in flight
    grid.sync();
    reduce_and_sgd(a, La + Lt, ntiles);
    if (blockIdx.x == 0) {
        // mean loss over the batch (fixed order) and the gradient channel's header
        __syncthreads();
        float part = 0.f;
        for (int r = threadIdx.x; r < a.rows; r += NT) part += __ldcg(a.rowloss + r);
        for (int o = 16; o > 0; o >>= 1) part += __shfl_down_sync(0xffffffffu, part, o);
        float* red = smem;
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = part;
        __syncthreads();
        if (threadIdx.x == 0) {
            float v = 0.f;
            for (int w = 0; w < NT / 32; ++w) v += red[w];
            *a.loss_out = v * inv_b;
            a.pub_hdr->k = a.k;
            a.pub_hdr->batch = a.batch;
            a.pub_hdr->version = a.version;
            __threadfence();
        }
    }
}

__global__ void __launch_bounds__(NT, 1) fused_passive_bwd_kernel(const FusedStepArgs a) {
    extern __shared__ __align__(16) float smem[];
    cg::grid_group grid = cg::this_grid();
    const int Lp = a.na;
    const int ldA = a.act_ld;
    float* ws = smem;
    float* acts = smem + a.w_floats;
    // slots: 0 = x_p; 1..Lp = f_p outputs (saved by the forward); Lp+1, Lp+2 = gradients
    auto act = [&](int i) { return acts + i * R * ldA; };
    float* g0 = act(Lp + 1);
    float* g1 = act(Lp + 2);
    float* red = act(Lp + 3);                   // K-split partial sums of tile_gemm
    if (threadIdx.x == 0 && a.chk_hdr->k != a.k) atomicOr(a.status, ST_VERSION);
    const FusedLayerArgs* P = a.L;
    const int ep = P[Lp - 1].out;
    const int ntiles = (a.rows + R - 1) / R;
    bool first = true;
    for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int r0 = tile * R;
        const int nr = min(R, a.rows - r0);
        float* part = a.part + (long long)tile * a.ptotal;
        __syncthreads();
        async_rows(act(0), ldA, a.x + (long long)r0 * a.ldx, a.ldx, (int)P[0].in_ld, nr);
        for (int l = 0; l < Lp; ++l)
            async_rows(act(l + 1), ldA, P[l].Y + (long long)r0 * P[l].ldy, P[l].ldy, (int)P[l].out_ld, nr);
        async_rows(g1, ldA, a.gradp + (long long)r0 * a.ldgp, a.ldgp, (int)P[Lp - 1].out_ld, nr);
        cp_commit();
        if (first) {
            // weights in the order the backward uses them: layer Lp-1 first
            for (int l = Lp - 1; l >= 1; --l) {
                stage_layer_weights(ws, P[l]);
                cp_commit();
            }
        }
        cp_wait_pending(first ? Lp - 1 : 0);
        for (int i = threadIdx.x; i < R * ep; i += NT) {                 // dz^p * [z^p > 0]
            const int r = i / ep, c = i - r * ep;
            const float v = act(Lp)[r * ldA + c] > 0.f ? g1[r * ldA + c] : 0.f;
            g0[r * ldA + c] = v;
            if (r < nr) P[Lp - 1].D[(long long)(r0 + r) * P[Lp - 1].ldd + c] = v;
        }
        float* gin = g0;
        float* gout = g1;
        for (int l = Lp - 1; l >= 0; --l) {
            __syncthreads();
            tile_partial(gin, ldA, act(l), ldA, P[l].out, P[l].in, part + P[l].poff);
            if (l > 0) {
                if (first) cp_wait_pending(l - 1);   // this layer's weights
                tile_dx(gin, ldA, P[l].out, ws + P[l].ws_off, P[l].ws_ld, P[l].in, act(l), ldA, gout, ldA,
                        P[l - 1].D + (long long)r0 * P[l - 1].ldd, P[l - 1].ldd, nr, red);
                float* t = gin;
                gin = gout;
                gout = t;
            }
        }
        first = false;
    }
    if (first) cp_wait_pending(0);
    grid.sync();
    reduce_and_sgd(a, Lp, ntiles);
}

template <typename K>
cudaError_t set_smem_attr(K kernel) {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFusedMaxSmem);
}

}  // namespace

cudaError_t launch_fused_passive_fwd(const FusedChainArgs& a, cudaStream_t s) {
    static cudaError_t attr = set_smem_attr(fused_passive_fwd_kernel);
    if (attr != cudaSuccess) return attr;
    const int ntiles = (a.rows + R - 1) / R;
    fused_passive_fwd_kernel<<<ntiles, NT, fused_smem_fwd(a.w_floats, a.act_ld), s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_fused_active(const FusedStepArgs& a, int grid, cudaStream_t s) {
    static cudaError_t attr = set_smem_attr(fused_active_kernel);
    if (attr != cudaSuccess) return attr;
    void* args[] = {(void*)&a};
    return cudaLaunchCooperativeKernel((const void*)fused_active_kernel, dim3(grid), dim3(NT), args,
                                       fused_smem_active(a.w_floats, a.act_ld, a.na, a.nt), s);
}

cudaError_t launch_fused_passive_bwd(const FusedStepArgs& a, int grid, cudaStream_t s) {
    static cudaError_t attr = set_smem_attr(fused_passive_bwd_kernel);
    if (attr != cudaSuccess) return attr;
    void* args[] = {(void*)&a};
    return cudaLaunchCooperativeKernel((const void*)fused_passive_bwd_kernel, dim3(grid), dim3(NT), args,
                                       fused_smem_pbwd(a.w_floats, a.act_ld, a.na), s);
}

cudaError_t fused_max_grid(int which, size_t smem, int* ctas) {
    int per_sm = 0, dev = 0, nsm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    const void* f = which == 0 ? (const void*)fused_active_kernel : (const void*)fused_passive_bwd_kernel;
    if (e == cudaSuccess) e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFusedMaxSmem);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, f, NT, smem);
    *ctas = per_sm * nsm;
    return e;
}

}  // namespace vfl
