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

constexpr int NT = kFusedThreads;     // 8 warps
constexpr int R = kFusedRows;

__device__ __forceinline__ void cp16(float* s, const float* g) {
    const unsigned sa = (unsigned)__cvta_generic_to_shared(s);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(sa), "l"(g) : "memory");
}

__device__ __forceinline__ void cp_wait_all() {
    asm volatile("cp.async.commit_group;\n" ::: "memory");
    asm volatile("cp.async.wait_group 0;\n" ::: "memory");
}

// n floats (n % 4 == 0; both ends 16-byte aligned), asynchronously
__device__ void async_copy(float* s, const float* g, long long n) {
    for (long long i = threadIdx.x; i < n / 4; i += NT) cp16(s + 4 * i, g + 4 * i);
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

__device__ void stage_layer_weights(float* ws, const FusedLayerArgs& L) {
    if (L.wts_off >= 0) async_copy(ws + L.wts_off, L.Wt, (long long)L.in * L.out_ld);
    if (L.ws_off >= 0) async_copy(ws + L.ws_off, L.W, (long long)L.out * L.in_ld);
}

// Y[r][c] = act(sum_k X[r][k] Wt[k][c] + b[c]) for the R = 16 rows of a tile.
// Each thread owns a 2-row x 4-column block (16-byte weight loads, 8 independent
// accumulators); Wt rows are zero beyond N.  To smem (ldy) and to global rows
// < nrows when yg != nullptr.
__device__ void tile_fwd(const float* xs, int ldx, int K, const float* wts, long long ldw,
                         const float* __restrict__ bias, int N, bool relu, float* ys, int ldy, float* yg,
                         long long ldyg, int nrows) {
    const int n4 = (N + 3) / 4;
    for (int u = threadIdx.x; u < (R / 2) * n4; u += NT) {
        const int cg = u % n4, r0 = 2 * (u / n4);
        const float* x0 = xs + r0 * ldx;
        const float* x1 = x0 + ldx;
        float a0[4] = {0.f, 0.f, 0.f, 0.f}, a1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
        for (int k = 0; k < K; ++k) {
            const float4 w = *reinterpret_cast<const float4*>(wts + k * ldw + 4 * cg);
            const float v0 = x0[k], v1 = x1[k];
            a0[0] = fmaf(v0, w.x, a0[0]); a0[1] = fmaf(v0, w.y, a0[1]);
            a0[2] = fmaf(v0, w.z, a0[2]); a0[3] = fmaf(v0, w.w, a0[3]);
            a1[0] = fmaf(v1, w.x, a1[0]); a1[1] = fmaf(v1, w.y, a1[1]);
            a1[2] = fmaf(v1, w.z, a1[2]); a1[3] = fmaf(v1, w.w, a1[3]);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int c = 4 * cg + j;
            if (c >= N) break;
            const float bv = bias[c];
            float y0 = a0[j] + bv, y1 = a1[j] + bv;
            if (relu) {
                y0 = fmaxf(y0, 0.f);
                y1 = fmaxf(y1, 0.f);
            }
            ys[r0 * ldy + c] = y0;
            ys[(r0 + 1) * ldy + c] = y1;
            if (yg) {
                if (r0 < nrows) yg[(long long)r0 * ldyg + c] = y0;
                if (r0 + 1 < nrows) yg[(long long)(r0 + 1) * ldyg + c] = y1;
            }
        }
    }
}

// dX[r][k] = sum_c dY[r][c] W[c][k], zeroed where prev[r][k] <= 0 (when prev is
// given); 2-row x 4-column blocks with 16-byte weight loads (W rows zero beyond
// K).  To smem and to global rows < nrows.
__device__ void tile_dx(const float* dys, int ldd, int N, const float* ws, long long ldw, int K, const float* prev,
                        int ldp, float* os, int ldo, float* og, long long ldog, int nrows) {
    const int k4 = (K + 3) / 4;
    for (int u = threadIdx.x; u < (R / 2) * k4; u += NT) {
        const int kg = u % k4, r0 = 2 * (u / k4);
        const float* d0 = dys + r0 * ldd;
        const float* d1 = d0 + ldd;
        float a0[4] = {0.f, 0.f, 0.f, 0.f}, a1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
        for (int c = 0; c < N; ++c) {
            const float4 w = *reinterpret_cast<const float4*>(ws + c * ldw + 4 * kg);
            const float v0 = d0[c], v1 = d1[c];
            a0[0] = fmaf(v0, w.x, a0[0]); a0[1] = fmaf(v0, w.y, a0[1]);
            a0[2] = fmaf(v0, w.z, a0[2]); a0[3] = fmaf(v0, w.w, a0[3]);
            a1[0] = fmaf(v1, w.x, a1[0]); a1[1] = fmaf(v1, w.y, a1[1]);
            a1[2] = fmaf(v1, w.z, a1[2]); a1[3] = fmaf(v1, w.w, a1[3]);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int k = 4 * kg + j;
            if (k >= K) break;
            float y0 = a0[j], y1 = a1[j];
            if (prev) {
                if (!(prev[r0 * ldp + k] > 0.f)) y0 = 0.f;
                if (!(prev[(r0 + 1) * ldp + k] > 0.f)) y1 = 0.f;
            }
            os[r0 * ldo + k] = y0;
            os[(r0 + 1) * ldo + k] = y1;
            if (og) {
                if (r0 < nrows) og[(long long)r0 * ldog + k] = y0;
                if (r0 + 1 < nrows) og[(long long)(r0 + 1) * ldog + k] = y1;
            }
        }
    }
}

// Partial gradient of one layer over the tile's rows, [W | b] flat:
// part[o*in + k] = sum_r D[r][o] X[r][k] and part[out*in + o] = sum_r D[r][o],
// in 4 x 4 register blocks fed by 16-byte loads.  Rows beyond the batch hold
// D = 0; columns past out / in in the tiles are never stored.
__device__ void tile_partial(const float* Ds, int ldd, const float* Xs, int ldx, int out, int in,
                             float* __restrict__ part) {
    const int o4 = (out + 3) / 4, i4 = (in + 3) / 4;
    for (int u = threadIdx.x; u < o4 * i4; u += NT) {
        const int ob = u / i4, ib = u - ob * i4;
        float acc[4][4] = {};
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const float4 d = *reinterpret_cast<const float4*>(Ds + r * ldd + 4 * ob);
            const float4 x = *reinterpret_cast<const float4*>(Xs + r * ldx + 4 * ib);
            const float dv[4] = {d.x, d.y, d.z, d.w}, xv[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(dv[i], xv[j], acc[i][j]);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int o = 4 * ob + i;
            if (o >= out) break;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int k = 4 * ib + j;
                if (k < in) part[(long long)o * in + k] = acc[i][j];
            }
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
            L.Wtc[k * L.out_ld + o] = w;
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
__global__ void __launch_bounds__(NT) fused_passive_fwd_kernel(const FusedChainArgs a) {
    extern __shared__ __align__(16) float smem[];
    float* ws = smem;
    float* buf0 = smem + a.w_floats;
    float* buf1 = buf0 + R * a.act_ld;
    for (int l = 0; l < a.nl; ++l) stage_layer_weights(ws, a.L[l]);
    const int ntiles = (a.rows + R - 1) / R;
    for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int r0 = tile * R;
        const int nr = min(R, a.rows - r0);
        __syncthreads();
        async_rows(buf0, a.act_ld, a.x + (long long)r0 * a.ldx, a.ldx, (int)a.L[0].in_ld, nr);
        cp_wait_all();
        __syncthreads();
        float* cur = buf0;
        float* nxt = buf1;
        for (int l = 0; l < a.nl; ++l) {
            const FusedLayerArgs& L = a.L[l];
            if (l) __syncthreads();
            tile_fwd(cur, a.act_ld, L.in, ws + L.wts_off, L.out_ld, L.b, L.out, true, nxt, a.act_ld,
                     L.Y + (long long)r0 * L.ldy, L.ldy, nr);
            float* t = cur;
            cur = nxt;
            nxt = t;
        }
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

__global__ void __launch_bounds__(NT) fused_active_kernel(const FusedStepArgs a) {
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
    if (threadIdx.x == 0 && a.chk_hdr->k != a.k) atomicOr(a.status, ST_VERSION);
    const FusedLayerArgs* A = a.L;
    const FusedLayerArgs* T = a.L + La;
    for (int l = 0; l < La + Lt; ++l) stage_layer_weights(ws, a.L[l]);
    const int ea = A[La - 1].out;
    const int ep = T[0].in - ea;
    const int nout = T[Lt - 1].out;
    const int ntiles = (a.rows + R - 1) / R;
    const float inv_b = 1.0f / (float)a.rows;
    for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int r0 = tile * R;
        const int nr = min(R, a.rows - r0);
        float* part = a.part + (long long)tile * a.ptotal;
        __syncthreads();
        async_rows(act(0), ldA, a.x + (long long)r0 * a.ldx, a.ldx, (int)A[0].in_ld, nr);
        async_rows(act(La + 1) + ea, ldA, a.zp + (long long)r0 * a.ldzp, a.ldzp, ep, nr);
        cp_wait_all();
        __syncthreads();
        for (int l = 0; l < La; ++l) {                                   // z^a = f_a(x^a)
            if (l) __syncthreads();
            tile_fwd(act(l), ldA, A[l].in, ws + A[l].wts_off, A[l].out_ld, A[l].b, A[l].out, true, act(l + 1), ldA,
                     A[l].Y + (long long)r0 * A[l].ldy, A[l].ldy, nr);
        }
        __syncthreads();
        for (int i = threadIdx.x; i < R * ea; i += NT) {                 // [z^a | z^p]
            const int r = i / ea, c = i - r * ea;
            act(La + 1)[r * ldA + c] = act(La)[r * ldA + c];
        }
        for (int l = 0; l < Lt; ++l) {                                   // y_hat = g(z^a, z^p)
            __syncthreads();
            tile_fwd(act(La + 1 + l), ldA, T[l].in, ws + T[l].wts_off, T[l].out_ld, T[l].b, T[l].out, l < Lt - 1,
                     act(La + 2 + l), ldA, T[l].Y + (long long)r0 * T[l].ldy, T[l].ldy, nr);
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
                tile_dx(gin, ldA, T[l].out, ws + T[l].ws_off, T[l].in_ld, T[l].in, act(La + 1 + l), ldA, gout, ldA,
                        T[l - 1].D + (long long)r0 * T[l - 1].ldd, T[l - 1].ldd, nr);
            else
                tile_dx(gin, ldA, T[l].out, ws + T[l].ws_off, T[l].in_ld, T[l].in, nullptr, 0, gout, ldA, nullptr, 0,
                        nr);
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
                tile_dx(gin, ldA, A[l].out, ws + A[l].ws_off, A[l].in_ld, A[l].in, act(l), ldA, gout, ldA,
                        A[l - 1].D + (long long)r0 * A[l - 1].ldd, A[l - 1].ldd, nr);
                float* t = gin;
                gin = gout;
                gout = t;
            }
        }
    }
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

__global__ void __launch_bounds__(NT) fused_passive_bwd_kernel(const FusedStepArgs a) {
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
    if (threadIdx.x == 0 && a.chk_hdr->k != a.k) atomicOr(a.status, ST_VERSION);
    const FusedLayerArgs* P = a.L;
    for (int l = 1; l < Lp; ++l) stage_layer_weights(ws, P[l]);
    const int ep = P[Lp - 1].out;
    const int ntiles = (a.rows + R - 1) / R;
    for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int r0 = tile * R;
        const int nr = min(R, a.rows - r0);
        float* part = a.part + (long long)tile * a.ptotal;
        __syncthreads();
        async_rows(act(0), ldA, a.x + (long long)r0 * a.ldx, a.ldx, (int)P[0].in_ld, nr);
        for (int l = 0; l < Lp; ++l)
            async_rows(act(l + 1), ldA, P[l].Y + (long long)r0 * P[l].ldy, P[l].ldy, (int)P[l].out_ld, nr);
        async_rows(g1, ldA, a.gradp + (long long)r0 * a.ldgp, a.ldgp, (int)P[Lp - 1].out_ld, nr);
        cp_wait_all();
        __syncthreads();
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
                tile_dx(gin, ldA, P[l].out, ws + P[l].ws_off, P[l].in_ld, P[l].in, act(l), ldA, gout, ldA,
                        P[l - 1].D + (long long)r0 * P[l - 1].ldd, P[l - 1].ldd, nr);
                float* t = gin;
                gin = gout;
                gout = t;
            }
        }
    }
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
