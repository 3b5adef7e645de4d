// SIMT kernels of the split-VFL step: the fp32 GEMM used for fp32 contexts and
// for narrow layers, the fused loss, DP clip+noise, ReLU mask, fused SGD, batched
// bias column sums, the parameter-server average, channel headers (behind a DP
// kernel; otherwise the GEMMs carry them) and data casts.
#include <algorithm>

#include "vfl_kernels.cuh"
#include "vfl_philox.cuh"
#include "vfl_pdl.cuh"

namespace vfl {

namespace {

__device__ __forceinline__ float ldf(const float* p) { return *p; }
__device__ __forceinline__ float ldf(const __nv_bfloat16* p) { return __bfloat162float(*p); }

__device__ __forceinline__ void stf(void* base, long long idx, int bf16, float v) {
    if (bf16)
        static_cast<__nv_bfloat16*>(base)[idx] = __float2bfloat16_rn(v);
    else
        static_cast<float*>(base)[idx] = v;
}

__device__ __forceinline__ float ldany(const void* base, long long idx, int bf16) {
    return bf16 ? __bfloat162float(static_cast<const __nv_bfloat16*>(base)[idx])
                : static_cast<const float*>(base)[idx];
}

constexpr int BM = 64, BN = 64, BK = 16, NT = 256;

template <typename TA, typename TB, typename TM>
__global__ void __launch_bounds__(NT) gemm_simt_kernel(const GemmArgs g) {
    pdl_entry();
    header_check(g.hdr);
    __shared__ float As[BK][BM + 1];
    __shared__ float Bs[BK][BN + 1];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int m0 = blockIdx.x * BM, n0 = blockIdx.y * BN;
    const int kb = blockIdx.z * g.kchunk;
    const int ke = min(g.K, kb + g.kchunk);
    const TA* A = static_cast<const TA*>(g.A);
    const TA* A2 = static_cast<const TA*>(g.A2);
    const TB* B = static_cast<const TB*>(g.B);
    float acc[4][4] = {};
    double bsum[4] = {};        // db partials in fp64: their per-row terms largely cancel
    const bool want_bsum = g.mode == GEMM_DW && blockIdx.y == 0 && tx == 0 && g.Pb != nullptr;

    for (int k0 = kb; k0 < ke; k0 += BK) {
        for (int e = threadIdx.x; e < BM * BK; e += NT) {
            int mm, kk;
            if (g.a_cs == 1) { mm = e / BK; kk = e % BK; } else { kk = e / BM; mm = e % BM; }
            const int m = m0 + mm, k = k0 + kk;
            float v = 0.f;
            if (m < g.M && k < ke) {
                if (A2 != nullptr && k >= g.ka)
                    v = ldf(A2 + (long long)m * g.a2_rs + (long long)(k - g.ka) * g.a_cs);
                else
                    v = ldf(A + (long long)m * g.a_rs + (long long)k * g.a_cs);
            }
            As[kk][mm] = v;
        }
        for (int e = threadIdx.x; e < BN * BK; e += NT) {
            int nn, kk;
            if (g.b_cs == 1) { nn = e / BK; kk = e % BK; } else { kk = e / BN; nn = e % BN; }
            const int n = n0 + nn, k = k0 + kk;
            float v = 0.f;
            if (n < g.N && k < ke) v = ldf(B + (long long)n * g.b_rs + (long long)k * g.b_cs);
            Bs[kk][nn] = v;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < BK; ++kk) {
            float av[4], bv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) av[i] = As[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) bv[j] = Bs[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
                if (want_bsum) bsum[i] += av[i];
            }
        }
        __syncthreads();
    }

#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int m = m0 + ty * 4 + i;
        if (m >= g.M) continue;
        if (want_bsum) g.Pb[(long long)blockIdx.z * g.pb_stride + m] = (float)bsum[i];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int n = n0 + tx * 4 + j;
            if (n >= g.N) continue;
            float v = acc[i][j];
            if (g.mode == GEMM_FWD) {
                if (g.bias) v += g.bias[n];
                if (g.relu) v = fmaxf(v, 0.f);
                stf(g.C, (long long)m * g.ldc + n, g.c_bf16, v);
            } else if (g.mode == GEMM_DX) {
                if (n < g.n_split) {
                    if (g.mask1 && !(ldf(static_cast<const TM*>(g.mask1) + (long long)m * g.mask1_ld + n) > 0.f))
                        v = 0.f;
                    stf(g.C, (long long)m * g.ldc + n, g.c_bf16, v);
                } else {
                    const int n2 = n - g.n_split;
                    if (g.mask2 && !(ldf(static_cast<const TM*>(g.mask2) + (long long)m * g.mask2_ld + n2) > 0.f))
                        v = 0.f;
                    stf(g.C2, (long long)m * g.ldc2 + n2, g.c2_bf16, v);
                }
            } else {
                g.P[(long long)blockIdx.z * g.p_stride + (long long)m * g.ldc + n] = v;
            }
        }
    }
    header_publish(g.hdr);
}

// Every kernel of the library asks for the shared-memory-heavy split of the SM's L1 / shared storage that
// the tcgen05 and fused kernels need: kernels of both kinds alternate within a step, and an SM whose split
// changes between two kernels has to drain before the next one starts.  Set once per kernel, on its first
// launch.
template <typename F>
inline bool prefer_shared_split(F* kernel) {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                (int)cudaSharedmemCarveoutMaxShared) == cudaSuccess;
}
#define SHARED_SPLIT(k)                                          \
    do {                                                         \
        static const bool split_set_ = prefer_shared_split(k);  \
        (void)split_set_;                                        \
    } while (0)

template <typename TA, typename TB>
cudaError_t gemm_dispatch_mask(const GemmArgs& g, int mask_bf16, dim3 grid, cudaStream_t s) {
    if (mask_bf16) {
        SHARED_SPLIT((gemm_simt_kernel<TA, TB, __nv_bfloat16>));
        gemm_simt_kernel<TA, TB, __nv_bfloat16><<<grid, NT, 0, s>>>(g);
    } else {
        SHARED_SPLIT((gemm_simt_kernel<TA, TB, float>));
        gemm_simt_kernel<TA, TB, float><<<grid, NT, 0, s>>>(g);
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Loss (BCE in logit form / softmax CE), one block, fixed-order reduction.
// ---------------------------------------------------------------------------
constexpr int LOSS_NT = 1024;

__global__ void __launch_bounds__(LOSS_NT) loss_kernel(const float* __restrict__ logits, const int* __restrict__ y,
                                                        int rows, int n_out, int kind, float* __restrict__ ds,
                                                        float* __restrict__ loss_out, float* loss_host) {
    pdl_entry();
    __shared__ float red[LOSS_NT / 32];
    const float inv_b = 1.0f / (float)rows;
    float part = 0.f;
    for (int r = threadIdx.x; r < rows; r += LOSS_NT) {
        const float* s = logits + (long long)r * n_out;
        float* d = ds + (long long)r * n_out;
        const int label = y[r];
        if (kind == VFL_LOSS_BCE) {
            const float x = s[0];
            const float yf = (float)label;
            part += fmaxf(x, 0.f) - x * yf + log1pf(expf(-fabsf(x)));
            const float sig = 1.0f / (1.0f + expf(-x));
            d[0] = (sig - yf) * inv_b;
        } else {
            float m = s[0];
            for (int j = 1; j < n_out; ++j) m = fmaxf(m, s[j]);
            float z = 0.f;
            for (int j = 0; j < n_out; ++j) z += expf(s[j] - m);
            part += logf(z) + m - s[label];
            const float iz = 1.0f / z;
            for (int j = 0; j < n_out; ++j) {
                const float p = expf(s[j] - m) * iz - (j == label ? 1.f : 0.f);
                d[j] = p * inv_b;
            }
        }
    }
    for (int o = 16; o > 0; o >>= 1) part += __shfl_down_sync(0xffffffffu, part, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = part;
    __syncthreads();
    if (threadIdx.x < 32) {
        float v = red[threadIdx.x];
        for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
        if (threadIdx.x == 0) {
            *loss_out = v * inv_b;
            if (loss_host) *loss_host = v * inv_b;
        }
    }
}

// ---------------------------------------------------------------------------
// Output layer + loss for the bf16 path (see HeadArgs).  256 threads, kHeadRows rows per block.
// Phase 0 stages W, the block's rows of h and their labels in shared memory with every load in
// flight at once.  Phase 1 gives warp w the rows w, w+8, ...; lane l holds inputs [8l, 8l+8) of a
// row, and W sits lane-minor (element (j, 8l+e) at (8j+e)*32 + l) so the warp's reads of it hit 32
// banks.  Phase 2 gives thread t the inputs [8 (t mod 32), +8) of outputs j = t/32, t/32 + 8.
constexpr int HEAD_NT = 256;
static_assert(kHeadMaxK == 32 * 8 && kHeadMaxOut <= 2 * (HEAD_NT / 32), "head thread map");

// NOUT: the output width the kernel is compiled for (1 for the BCE head, kHeadMaxOut otherwise); the
// arrays sized by it stay in registers, and the single-logit kernel needs far fewer of them.
template <int NOUT>
__global__ void __launch_bounds__(HEAD_NT) head_kernel(const HeadArgs a) {
    pdl_entry();
    __shared__ float Ws[NOUT * kHeadMaxK];          // lane-minor: (j, 8l + e) at (8j + e) * 32 + l
    __shared__ __align__(16) __nv_bfloat16 hs[kHeadRows * kHeadMaxK];
    __shared__ float dss[kHeadRows * NOUT];
    __shared__ int ys[kHeadRows];
    __shared__ float wloss[HEAD_NT / 32];
    __shared__ bool last;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int K = a.K, nout = a.nout;
    const int r0 = blockIdx.x * kHeadRows, nr = min(kHeadRows, a.rows - r0);
    const float inv_b = 1.0f / (float)a.rows;
    const __nv_bfloat16* W = static_cast<const __nv_bfloat16*>(a.W);
    const __nv_bfloat16* Hg = static_cast<const __nv_bfloat16*>(a.h);
    // phase 0: W, the rows (zero past nr and past K) and the labels
    for (int i = tid; i < nout * K; i += HEAD_NT) {
        const int j = i / K, k = i - j * K;
        Ws[(j * 8 + (k & 7)) * 32 + (k >> 3)] = __bfloat162float(W[(long long)j * a.ldw + k]);
    }
    for (int i = tid; i < kHeadRows * (kHeadMaxK / 8); i += HEAD_NT) {
        const int r = i >> 5, c = (i & 31) * 8;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (r < nr && c < K) v = *reinterpret_cast<const uint4*>(Hg + (long long)(r0 + r) * a.ldh + c);
        *reinterpret_cast<uint4*>(hs + r * kHeadMaxK + c) = v;
    }
    if (tid < kHeadRows) ys[tid] = tid < nr ? a.y[r0 + tid] : 0;
    __syncthreads();
    const bool kin = lane * 8 < K;
    float wl = 0.f;                                     // this warp's rows' loss, in row order
    for (int r = warp; r < kHeadRows; r += HEAD_NT / 32) {
        float hk[8];
        const uint4 raw = *reinterpret_cast<const uint4*>(hs + r * kHeadMaxK + lane * 8);
        const __nv_bfloat16* hb = reinterpret_cast<const __nv_bfloat16*>(&raw);
#pragma unroll
        for (int e = 0; e < 8; ++e) hk[e] = __bfloat162float(hb[e]);
        float sv[NOUT], dv[NOUT];
#pragma unroll
        for (int j = 0; j < NOUT; ++j) {
            if (j < nout) {
                float p = 0.f;
                const float* w = Ws + j * kHeadMaxK + lane;
#pragma unroll
                for (int e = 0; e < 8; ++e) p = fmaf(hk[e], kin ? w[e * 32] : 0.f, p);
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) p += __shfl_xor_sync(0xffffffffu, p, o);
                sv[j] = p + a.b[j];
            }
        }
        float li = 0.f;
        if (r < nr) {
            const int yl = ys[r];
            if (a.loss == VFL_LOSS_BCE) {
                const float x = sv[0];
                li = fmaxf(x, 0.f) - x * (float)yl + log1pf(expf(-fabsf(x)));
                dv[0] = (1.0f / (1.0f + expf(-x)) - (float)yl) * inv_b;
            } else {
                float m = sv[0];
#pragma unroll
                for (int j = 1; j < NOUT; ++j)
                    if (j < nout) m = fmaxf(m, sv[j]);
                float z = 0.f;
#pragma unroll
                for (int j = 0; j < NOUT; ++j)
                    if (j < nout) z += expf(sv[j] - m);
                float sy = 0.f;
#pragma unroll
                for (int j = 0; j < NOUT; ++j)
                    if (j < nout && j == yl) sy = sv[j];
                li = logf(z) + m - sy;
                const float iz = 1.0f / z;
#pragma unroll
                for (int j = 0; j < NOUT; ++j)
                    if (j < nout) dv[j] = (expf(sv[j] - m) * iz - (j == yl ? 1.f : 0.f)) * inv_b;
            }
            wl += li;
            if (lane < nout) {
                float sl = 0.f, dl = 0.f;
#pragma unroll
                for (int j = 0; j < NOUT; ++j)
                    if (j == lane) { sl = sv[j]; dl = dv[j]; }
                a.logits[(long long)(r0 + r) * nout + lane] = sl;
                a.ds[(long long)(r0 + r) * nout + lane] = dl;
            }
        } else {
#pragma unroll
            for (int j = 0; j < NOUT; ++j) dv[j] = 0.f;
        }
        if (lane < nout) {
            float dl = 0.f;
#pragma unroll
            for (int j = 0; j < NOUT; ++j)
                if (j == lane) dl = dv[j];
            dss[r * NOUT + lane] = dl;
        }
        if (r < nr && kin) {                            // hidden layer's d(pre-activation), bf16
            __align__(16) __nv_bfloat16 ob[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                float g = 0.f;
#pragma unroll
                for (int j = 0; j < NOUT; ++j)
                    if (j < nout) g = fmaf(dv[j], Ws[(j * 8 + e) * 32 + lane], g);
                ob[e] = __float2bfloat16_rn(hk[e] > 0.f ? g : 0.f);
            }
            *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.dh) + (long long)(r0 + r) * a.lddh + lane * 8) =
                *reinterpret_cast<const uint4*>(ob);
        }
    }
    if (lane == 0) wloss[warp] = wl;
    __syncthreads();
    // partial dW and db of this block, rows in order
    {
        const int kc = (tid & 31) * 8;
        const int j0 = tid >> 5;
        if (kc < K) {
#pragma unroll
            for (int jj = 0; jj < 2; ++jj) {
                const int j = j0 + jj * (HEAD_NT / 32);
                if (j >= nout) break;
                float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
                for (int r = 0; r < nr; ++r) {
                    const float d = dss[r * NOUT + j];
                    const uint4 raw = *reinterpret_cast<const uint4*>(hs + r * kHeadMaxK + kc);
                    const __nv_bfloat16* hb = reinterpret_cast<const __nv_bfloat16*>(&raw);
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[e] = fmaf(d, __bfloat162float(hb[e]), acc[e]);
                }
                float* pw = a.pW + blockIdx.x * a.pw_stride + (long long)j * K + kc;
#pragma unroll
                for (int e = 0; e < 8; ++e) pw[e] = acc[e];
            }
        }
        if (tid < nout) {
            float sb = 0.f;
            for (int r = 0; r < nr; ++r) sb += dss[r * NOUT + tid];
            a.pb[blockIdx.x * a.pb_stride + tid] = sb;
        }
    }
    // the step's mean loss: block sums in block order, by the last block to finish
    if (tid == 0) {
        float v = 0.f;
        for (int w = 0; w < HEAD_NT / 32; ++w) v += wloss[w];
        a.blk_loss[blockIdx.x] = v;
        __threadfence();
        last = atomicAdd(a.counter, 1) == (int)gridDim.x - 1;
    }
    __syncthreads();
    if (last) {
        // thread t sums blocks t, t + HEAD_NT, ... in order, then a fixed shuffle tree and the warps in order
        __threadfence();
        float v = 0.f;
        for (int bb = tid; bb < (int)gridDim.x; bb += HEAD_NT) v += __ldcg(a.blk_loss + bb);
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) wloss[warp] = v;
        __syncthreads();
        if (tid == 0) {
            float t = 0.f;
            for (int w = 0; w < HEAD_NT / 32; ++w) t += wloss[w];
            *a.loss_out = t * inv_b;
            if (a.loss_host) *a.loss_host = t * inv_b;
            *a.counter = 0;
            __threadfence();
        }
    }
}

// ---------------------------------------------------------------------------
// DP: per-row clip of the per-sample gradient B*dz to norm C, plus sigma*C*N(0,1).
// ---------------------------------------------------------------------------
constexpr int DP_NT = 256;
constexpr int DP_ROWS = DP_NT / 32;            // one warp per row

// Sum over the warp's lanes in a fixed shuffle order.
__device__ __forceinline__ float warp_sum(float v) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Four consecutive values of a row (fp32 or bf16) starting at column c (c + 4 <= e, 16- / 8-byte aligned).
__device__ __forceinline__ void ld4(const void* base, long long idx, int bf16, float v[4]) {
    if (bf16) {
        const uint2 w = *reinterpret_cast<const uint2*>(static_cast<const __nv_bfloat16*>(base) + idx);
        const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w.x));
        const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w.y));
        v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
    } else {
        const float4 f = *reinterpret_cast<const float4*>(static_cast<const float*>(base) + idx);
        v[0] = f.x; v[1] = f.y; v[2] = f.z; v[3] = f.w;
    }
}

__device__ __forceinline__ void st4(void* base, long long idx, int bf16, const float v[4]) {
    if (bf16) {
        const __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]), b = __floats2bfloat162_rn(v[2], v[3]);
        uint2 w;
        w.x = *reinterpret_cast<const uint32_t*>(&a);
        w.y = *reinterpret_cast<const uint32_t*>(&b);
        *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(base) + idx) = w;
    } else {
        *reinterpret_cast<float4*>(static_cast<float*>(base) + idx) = make_float4(v[0], v[1], v[2], v[3]);
    }
}

// DP on the published gradient (App. C reading): per row g = B_k dz, factor = min(1, C / ||g||),
// out = (g factor + sigma C N(0,1)) / B_k.  One warp per row; lane l takes the 4-column groups
// q = l, l + 32, ... (the Philox block of group q gives its four normals).  Rows are 16-byte aligned
// (leading dims are multiples of 8 elements).
__global__ void __launch_bounds__(DP_NT) dp_kernel(const float* __restrict__ in, long long ld_in, void* out,
                                                    long long ld_out, int out_bf16, int rows, int e, float clip,
                                                    float sigma, unsigned long long seed, long long k, float bk) {
    pdl_entry();
    const int lane = threadIdx.x & 31;
    const int r = blockIdx.x * DP_ROWS + (threadIdx.x >> 5);
    if (r >= rows) return;
    const float* row = in + (long long)r * ld_in;
    float ss = 0.f;
    for (int q = lane; 4 * q < e; q += 32) {
        float v[4];
        if (4 * q + 4 <= e) {
            ld4(row, 4 * q, 0, v);
        } else {
            for (int j = 0; j < 4; ++j) v[j] = 4 * q + j < e ? row[4 * q + j] : 0.f;
        }
        for (int j = 0; j < 4; ++j) {
            const float gv = v[j] * bk;
            ss = fmaf(gv, gv, ss);
        }
    }
    const float norm = sqrtf(warp_sum(ss));
    const float factor = norm > clip ? clip / norm : 1.0f;
    const uint2 key = make_uint2((unsigned)(seed & 0xFFFFFFFFull), (unsigned)(seed >> 32));
    const float scale = sigma * clip;
    for (int q = lane; 4 * q < e; q += 32) {
        float z[4], v[4];
        dp_normals4(q, r, k, 0x4450u, key, z);
        const bool whole = 4 * q + 4 <= e;
        if (whole) {
            ld4(row, 4 * q, 0, v);
        } else {
            for (int j = 0; j < 4; ++j) v[j] = 4 * q + j < e ? row[4 * q + j] : 0.f;
        }
        for (int j = 0; j < 4; ++j) v[j] = (v[j] * bk * factor + scale * z[j]) / bk;
        if (whole) {
            st4(out, (long long)r * ld_out + 4 * q, out_bf16, v);
        } else {
            for (int j = 0; j < 4 && 4 * q + j < e; ++j) stf(out, (long long)r * ld_out + 4 * q + j, out_bf16, v[j]);
        }
    }
}

// DP on the published embedding (App. C): per row c = min(1, C / ||z||) (1 for a zero row), the
// payload c z + sigma C N(0,1) (tag 0x4445) in the compute dtype, and c kept for the backward.
// One warp per row, as dp_kernel.
__global__ void __launch_bounds__(DP_NT) dp_emb_kernel(const void* z, long long ld, int bf16, void* out,
                                                        float* __restrict__ scale_out, int rows, int e, float clip,
                                                        float sigma, unsigned long long seed, long long k) {
    pdl_entry();
    const int lane = threadIdx.x & 31;
    const int r = blockIdx.x * DP_ROWS + (threadIdx.x >> 5);
    if (r >= rows) return;
    const long long base = (long long)r * ld;
    float ss = 0.f;
    for (int q = lane; 4 * q < e; q += 32) {
        float v[4];
        if (4 * q + 4 <= e) {
            ld4(z, base + 4 * q, bf16, v);
        } else {
            for (int j = 0; j < 4; ++j) v[j] = 4 * q + j < e ? ldany(z, base + 4 * q + j, bf16) : 0.f;
        }
        for (int j = 0; j < 4; ++j) ss = fmaf(v[j], v[j], ss);
    }
    const float norm = sqrtf(warp_sum(ss));
    const float factor = norm > clip ? clip / norm : 1.0f;
    if (lane == 0) scale_out[r] = factor;
    const uint2 key = make_uint2((unsigned)(seed & 0xFFFFFFFFull), (unsigned)(seed >> 32));
    const float noise = sigma * clip;
    for (int q = lane; 4 * q < e; q += 32) {
        float xi[4] = {0.f, 0.f, 0.f, 0.f}, v[4];
        if (noise != 0.f) dp_normals4(q, r, k, 0x4445u, key, xi);
        const bool whole = 4 * q + 4 <= e;
        if (whole) {
            ld4(z, base + 4 * q, bf16, v);
        } else {
            for (int j = 0; j < 4; ++j) v[j] = 4 * q + j < e ? ldany(z, base + 4 * q + j, bf16) : 0.f;
        }
        for (int j = 0; j < 4; ++j) v[j] = fmaf(v[j], factor, noise * xi[j]);
        if (whole) {
            st4(out, base + 4 * q, bf16, v);
        } else {
            for (int j = 0; j < 4 && 4 * q + j < e; ++j) stf(out, base + 4 * q + j, bf16, v[j]);
        }
    }
}

// out = g * [z > 0], with g first scaled by rs[row] when rs is given (rounded to T); each thread takes
// four consecutive columns of one row (rows are 16-byte aligned: ld is a multiple of 8 elements)
template <typename T>
__global__ void relu_mask_kernel(const T* __restrict__ g, const T* __restrict__ z, T* __restrict__ out,
                                 long long ld, int rows, int e, const float* __restrict__ rs, const HeaderOps hdr) {
    pdl_entry();
    header_check(hdr);
    const int bf = sizeof(T) == 2;
    const int gq = (e + 3) / 4;
    const int n = rows * gq;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        const int r = i / gq, c = (i - r * gq) * 4;
        const long long idx = (long long)r * ld + c;
        if (c + 4 <= e) {
            float gv[4], zv[4], o[4];
            ld4(g, idx, bf, gv);
            ld4(z, idx, bf, zv);
            for (int j = 0; j < 4; ++j) {
                float v = gv[j];
                if (rs) v = (float)T(rs[r] * v);
                o[j] = zv[j] > 0.f ? v : 0.f;
            }
            st4(out, idx, bf, o);
        } else {
            for (int j = 0; c + j < e; ++j)
                out[idx + j] = ldf(z + idx + j) > 0.f ? (rs ? T(rs[r] * ldf(g + idx + j)) : g[idx + j]) : T(0.f);
        }
    }
}

// ---------------------------------------------------------------------------
// SGD (Eq. 2): master -= lr * sum_z partial[z]; write the new version's copy.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void sgd_apply_w(const SgdArgs& a, const SgdLayer& L, int r, int c, float g) {
    const long long idx = (long long)r * L.in + c;
    const float w = L.W[idx] - a.lr * g;
    L.W[idx] = w;
    stf(L.cW, (long long)r * L.in_ld + c, a.c_bf16, w);
}

__device__ __forceinline__ void sgd_apply_b(const SgdArgs& a, const SgdLayer& L, int j, double g) {
    const float b = L.b[j] - a.lr * (float)g;
    L.b[j] = b;
    L.cb[j] = b;
}

// SGD (Eq. 2) for every layer of a party: layer blockIdx.y, its out * in weights then its out biases
// spread over the x blocks.  A layer with few partials takes one thread per parameter (partials summed in
// order; the bias partials in fp64, they largely cancel); one with many (a folded output layer's
// per-block partials) one warp per parameter: lane l sums partials l, l + 32, ... in order, then a fixed
// shuffle tree.
__global__ void __launch_bounds__(256) sgd_kernel(const SgdArgs a) {
    pdl_entry();
    const SgdLayer& L = a.L[blockIdx.y];
    const int nw = L.out * L.in, np = nw + L.out;
    if (L.nsplit < 16 && L.nsplit_b < 16 && (L.in & 3) == 0 && (L.in_ld & 3) == 0) {
        // rows of a multiple of four: four weights a thread (16-byte master and partial loads, 16-byte
        // master stores, 8- or 16-byte copy stores), the same fp32 sums in partial order
        const int nw4 = nw >> 2;
        const long long st4 = L.pW_stride >> 2;
        const float4* __restrict__ pW4 = reinterpret_cast<const float4*>(L.pW);
        float4* __restrict__ W4 = reinterpret_cast<float4*>(L.W);
        const int t0 = blockIdx.x * blockDim.x + threadIdx.x, nt = gridDim.x * blockDim.x;
        for (int i = t0; i < nw4; i += nt) {
            float4 g = pW4[i];
            for (int z = 1; z < L.nsplit; ++z) {
                const float4 h = pW4[z * st4 + i];
                g.x += h.x; g.y += h.y; g.z += h.z; g.w += h.w;
            }
            float4 w = W4[i];
            w.x -= a.lr * g.x; w.y -= a.lr * g.y; w.z -= a.lr * g.z; w.w -= a.lr * g.w;
            W4[i] = w;
            const int r = (4 * i) / L.in, c = 4 * i - r * L.in;
            const long long o = (long long)r * L.in_ld + c;
            if (a.c_bf16) {
                const __nv_bfloat162 lo = __floats2bfloat162_rn(w.x, w.y), hi = __floats2bfloat162_rn(w.z, w.w);
                *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(L.cW) + o) =
                    make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi));
            } else {
                *reinterpret_cast<float4*>(static_cast<float*>(L.cW) + o) = w;
            }
        }
        for (int j = t0; j < L.out; j += nt) {
            double g = 0.0;
            for (int z = 0; z < L.nsplit_b; ++z) g += L.pb[z * L.pb_stride + j];
            sgd_apply_b(a, L, j, g);
        }
        return;
    }
    if (L.nsplit < 16 && L.nsplit_b < 16) {
        for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < np; i += gridDim.x * blockDim.x) {
            if (i < nw) {
                float g = 0.f;
                for (int z = 0; z < L.nsplit; ++z) g += L.pW[z * L.pW_stride + i];
                const int r = i / L.in;
                sgd_apply_w(a, L, r, i - r * L.in, g);
            } else {
                double g = 0.0;
                for (int z = 0; z < L.nsplit_b; ++z) g += L.pb[z * L.pb_stride + (i - nw)];
                sgd_apply_b(a, L, i - nw, g);
            }
        }
        return;
    }
    const int lane = threadIdx.x & 31;
    const int nwarps = gridDim.x * (blockDim.x / 32);
    for (int i = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); i < np; i += nwarps) {
        if (i < nw) {
            float g = 0.f;
            for (int z = lane; z < L.nsplit; z += 32) g += L.pW[z * L.pW_stride + i];
            for (int o = 16; o > 0; o >>= 1) g += __shfl_xor_sync(0xffffffffu, g, o);
            const int r = i / L.in;
            if (lane == 0) sgd_apply_w(a, L, r, i - r * L.in, g);
        } else {
            double g = 0.0;
            for (int z = lane; z < L.nsplit_b; z += 32) g += L.pb[z * L.pb_stride + (i - nw)];
            for (int o = 16; o > 0; o >>= 1) g += __shfl_xor_sync(0xffffffffu, g, o);
            if (lane == 0) sgd_apply_b(a, L, i - nw, g);
        }
    }
}

__global__ void __launch_bounds__(256) ps_average_kernel(const PsAvgLayer* __restrict__ tab, int n_layers,
                                                         long long total, int nrep, int c_bf16) {
    pdl_entry();
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        int l = 0;
        while (l + 1 < n_layers && i >= tab[l + 1].begin) ++l;
        const PsAvgLayer& L = tab[l];
        const long long idx = i - L.begin;
        const long long nw = (long long)L.out * L.in;
        if (idx < nw) {
            float acc = 0.f;
            for (int w = 0; w < nrep; ++w) acc += L.Wr[w][idx];
            const float v = __fdiv_rn(acc, (float)nrep);
            const long long r = idx / L.in, c = idx % L.in;
            for (int w = 0; w < nrep; ++w) {
                L.Wr[w][idx] = v;
                stf(L.cW[w], r * L.in_ld + c, c_bf16, v);
            }
        } else {
            const long long j = idx - nw;
            float acc = 0.f;
            for (int w = 0; w < nrep; ++w) acc += L.br[w][j];
            const float v = __fdiv_rn(acc, (float)nrep);
            for (int w = 0; w < nrep; ++w) {
                L.br[w][j] = v;
                L.cb[w][j] = v;
            }
        }
    }
}

__global__ void mark_dropped_kernel(float* loss, float* loss_host) {
    pdl_entry();
    const float nan = __int_as_float(0x7FC00000);
    *loss = nan;
    if (loss_host) *loss_host = nan;
}

__global__ void write_header_kernel(ChannelHeader* h, long long k, int batch, int version) {
    pdl_entry();
    h->k = k;
    h->batch = batch;
    h->version = version;
    __threadfence();
}

__global__ void check_header_kernel(const ChannelHeader* h, long long k, int* status) {
    pdl_entry();
    if (h->k != k) atomicOr(status, ST_VERSION);
}

// Bounded poll: gives up after max_iters reads and records ST_TIMEOUT.
__global__ void wait_header_kernel(const ChannelHeader* h, long long k, long long max_iters, int* status) {
    pdl_entry();
    const volatile long long* pk = &h->k;
    for (long long it = 0; it < max_iters; ++it) {
        if (*pk == k) return;
        __nanosleep(256);
    }
    atomicOr(status, ST_TIMEOUT);
}

__global__ void cast_rows_kernel(const float* __restrict__ src, int rows, int d, void* dst, long long ld, int bf16) {
    pdl_entry();
    const long long n = (long long)rows * ld;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        const long long r = i / ld, c = i % ld;
        const float v = c < d ? src[r * d + c] : 0.f;
        stf(dst, i, bf16, v);
    }
}

// One step's rows from host memory (read over the C2C link / PCIe as the kernel runs): element i of
// the padded passive rows, then of the padded active rows, then the labels.
// One party's block of rows [rows, d] fp32 (contiguous in host memory) into staging rows of ld elements
// (bf16 or fp32), padding columns zero.  Four consecutive values a thread when d is a multiple of 4 and
// the block is 16-byte aligned, four such groups loaded before any is stored (the loads cross the
// host link: as many as possible in flight).
__device__ __forceinline__ void stage_block(const float* __restrict__ h, int d, int rows, void* dst, long long ld,
                                            int bf16, int tid, int nthreads) {
    const int n = rows * d;
    if ((d & 3) == 0 && (reinterpret_cast<uintptr_t>(h) & 15) == 0 && (ld & 3) == 0) {
        const int nq = n / 4;
        constexpr int U = 4;
        for (int q0 = tid; q0 < nq; q0 += nthreads * U) {
            float4 v[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int q = q0 + u * nthreads;
                if (q < nq) v[u] = __ldcs(reinterpret_cast<const float4*>(h) + q);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int q = q0 + u * nthreads;
                if (q >= nq) break;
                const int f = 4 * q, r = f / d, c = f - r * d;
                const float vals[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
                if (bf16) {
                    const __nv_bfloat162 a = __floats2bfloat162_rn(vals[0], vals[1]), b = __floats2bfloat162_rn(vals[2], vals[3]);
                    uint2 w;
                    w.x = *reinterpret_cast<const uint32_t*>(&a);
                    w.y = *reinterpret_cast<const uint32_t*>(&b);
                    *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(dst) + (long long)r * ld + c) = w;
                } else {
                    *reinterpret_cast<float4*>(static_cast<float*>(dst) + (long long)r * ld + c) = v[u];
                }
            }
        }
    } else {
        for (int i = tid; i < n; i += nthreads) {
            const int r = i / d, c = i - r * d;
            stf(dst, (long long)r * ld + c, bf16, h[i]);
        }
    }
    // padding columns
    const int pad = (int)(ld - d);
    for (int i = tid; i < rows * pad; i += nthreads) {
        const int r = i / pad, c = d + (i - r * pad);
        stf(dst, (long long)r * ld + c, bf16, 0.f);
    }
}

// The same for bf16 host rows into a bf16 slot: 16-byte copies of eight elements where rows allow.
__device__ __forceinline__ void stage_block_b16(const uint16_t* __restrict__ h, int d, int rows, uint16_t* dst,
                                                long long ld, int tid, int nthreads) {
    const int n = rows * d;
    if ((d & 7) == 0 && (reinterpret_cast<uintptr_t>(h) & 15) == 0 && (ld & 7) == 0) {
        const int nq = n / 8;
        constexpr int U = 4;
        for (int q0 = tid; q0 < nq; q0 += nthreads * U) {
            uint4 v[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int q = q0 + u * nthreads;
                if (q < nq) v[u] = __ldcs(reinterpret_cast<const uint4*>(h) + q);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int q = q0 + u * nthreads;
                if (q >= nq) break;
                const int f = 8 * q, r = f / d, c = f - r * d;
                *reinterpret_cast<uint4*>(dst + (long long)r * ld + c) = v[u];
            }
        }
    } else {
        for (int i = tid; i < n; i += nthreads) {
            const int r = i / d, c = i - r * d;
            dst[(long long)r * ld + c] = h[i];
        }
    }
    const int pad = (int)(ld - d);
    for (int i = tid; i < rows * pad; i += nthreads) {
        const int r = i / pad, c = d + (i - r * pad);
        dst[(long long)r * ld + c] = 0;
    }
}

__global__ void stage_rows_b16_kernel(const uint16_t* __restrict__ hxp, int dp, const uint16_t* __restrict__ hxa,
                                      int da, const int* __restrict__ hy, int rows, uint16_t* xp, long long ld_p,
                                      uint16_t* xa, long long ld_a, int* __restrict__ y) {
    pdl_entry();
    const int tid = blockIdx.x * blockDim.x + threadIdx.x, nt = gridDim.x * blockDim.x;
    stage_block_b16(hxp, dp, rows, xp, ld_p, tid, nt);
    stage_block_b16(hxa, da, rows, xa, ld_a, tid, nt);
    for (int i = tid; i < rows; i += nt) y[i] = hy[i];
}

__global__ void stage_rows_kernel(const float* __restrict__ hxp, int dp, const float* __restrict__ hxa, int da,
                                  const int* __restrict__ hy, int rows, void* xp, long long ld_p, void* xa,
                                  long long ld_a, int* __restrict__ y, int bf16) {
    pdl_entry();
    const int tid = blockIdx.x * blockDim.x + threadIdx.x, nt = gridDim.x * blockDim.x;
    stage_block(hxp, dp, rows, xp, ld_p, bf16, tid, nt);
    stage_block(hxa, da, rows, xa, ld_a, bf16, tid, nt);
    for (int i = tid; i < rows; i += nt) y[i] = hy[i];
}

__global__ void to_f32_kernel(const void* src, long long ld, int rows, int cols, int bf16, float* dst) {
    pdl_entry();
    const long long n = (long long)rows * cols;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        const long long r = i / cols, c = i % cols;
        dst[i] = ldany(src, r * ld + c, bf16);
    }
}

// Blocks of a host-staging kernel: four per SM already pull the host link's full rate, and the step's compute
// kernels keep the rest of the SMs' warp slots.
constexpr int kStageBlocks = 152 * 4;

inline int grid_for(long long n, int nt) {
    long long b = (n + nt - 1) / nt;
    if (b < 1) b = 1;
    if (b > 152 * 16) b = 152 * 16;
    return (int)b;
}

}  // namespace

cudaError_t launch_gemm_simt(const GemmArgs& g, int a_bf16, int b_bf16, int mask_bf16, int nsplit, cudaStream_t s) {
    if (g.M <= 0 || g.N <= 0) return cudaSuccess;
    GemmArgs a = g;
    if (a.mode != GEMM_DW) {
        nsplit = 1;
        a.kchunk = a.K;
    }
    // DW: every one of the nsplit partials is written (zeros where its chunk is empty)
    if (nsplit < 1 || a.kchunk < 1) return cudaErrorInvalidValue;
    dim3 grid((a.M + BM - 1) / BM, (a.N + BN - 1) / BN, nsplit);
    if (a_bf16 && b_bf16) return gemm_dispatch_mask<__nv_bfloat16, __nv_bfloat16>(a, mask_bf16, grid, s);
    if (a_bf16) return gemm_dispatch_mask<__nv_bfloat16, float>(a, mask_bf16, grid, s);
    if (b_bf16) return gemm_dispatch_mask<float, __nv_bfloat16>(a, mask_bf16, grid, s);
    return gemm_dispatch_mask<float, float>(a, mask_bf16, grid, s);
}

cudaError_t launch_loss(const float* logits, const int* y, int rows, int n_out, int loss_kind, float* ds,
                        float* loss_out, float* loss_host, cudaStream_t s) {
    SHARED_SPLIT(loss_kernel);
    loss_kernel<<<1, LOSS_NT, 0, s>>>(logits, y, rows, n_out, loss_kind, ds, loss_out, loss_host);
    return cudaGetLastError();
}

cudaError_t launch_head(const HeadArgs& a, cudaStream_t s) {
    if (a.rows < 1 || a.nout < 1 || a.nout > kHeadMaxOut || a.K < 8 || a.K > kHeadMaxK || (a.K & 7) ||
        a.nblk < head_blocks(a.rows))
        return cudaErrorInvalidValue;
    if (a.nout == 1) {
        SHARED_SPLIT(head_kernel<1>);
        head_kernel<1><<<a.nblk, HEAD_NT, 0, s>>>(a);
    } else {
        SHARED_SPLIT(head_kernel<kHeadMaxOut>);
        head_kernel<kHeadMaxOut><<<a.nblk, HEAD_NT, 0, s>>>(a);
    }
    return cudaGetLastError();
}

cudaError_t launch_dp(const float* in, long long ld_in, void* out, long long ld_out, int out_bf16, int rows, int e,
                      float clip, float sigma, unsigned long long seed, long long k, cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    SHARED_SPLIT(dp_kernel);
    dp_kernel<<<(rows + DP_ROWS - 1) / DP_ROWS, DP_NT, 0, s>>>(in, ld_in, out, ld_out, out_bf16, rows, e, clip, sigma,
                                                               seed, k, (float)rows);
    return cudaGetLastError();
}

cudaError_t launch_relu_mask(const void* g, const void* z, void* out, long long ld, int rows, int e, int bf16,
                             const float* row_scale, const HeaderOps& hdr, cudaStream_t s) {
    const int nb = grid_for((long long)rows * ((e + 3) / 4), 256);
    if (bf16) {
        SHARED_SPLIT(relu_mask_kernel<__nv_bfloat16>);
        relu_mask_kernel<__nv_bfloat16><<<nb, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(g),
                                                           static_cast<const __nv_bfloat16*>(z),
                                                           static_cast<__nv_bfloat16*>(out), ld, rows, e, row_scale,
                                                           hdr);
    } else {
        SHARED_SPLIT(relu_mask_kernel<float>);
        relu_mask_kernel<float><<<nb, 256, 0, s>>>(static_cast<const float*>(g), static_cast<const float*>(z),
                                                   static_cast<float*>(out), ld, rows, e, row_scale, hdr);
    }
    return cudaGetLastError();
}

cudaError_t launch_dp_emb(const void* z, long long ld, int bf16, void* out, float* scale_out, int rows, int e,
                          float clip, float sigma, unsigned long long seed, long long k, cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    SHARED_SPLIT(dp_emb_kernel);
    dp_emb_kernel<<<(rows + DP_ROWS - 1) / DP_ROWS, DP_NT, 0, s>>>(z, ld, bf16, out, scale_out, rows, e, clip, sigma,
                                                                   seed, k);
    return cudaGetLastError();
}

cudaError_t launch_sgd(const SgdArgs& a, cudaStream_t s) {
    if (a.n_layers < 1) return cudaSuccess;
    // enough x blocks for the largest layer (a warp per parameter where partials are many), within a
    // few waves of the SMs over all layers
    long long most = 1;
    for (int l = 0; l < a.n_layers; ++l) {
        const long long np = (long long)a.L[l].out * a.L[l].in + a.L[l].out;
        const bool warp = a.L[l].nsplit >= 16 || a.L[l].nsplit_b >= 16;
        most = std::max(most, warp ? np * 32 : np);
    }
    const long long bx = std::min<long long>((most + 255) / 256, std::max(1, 152 * 8 / a.n_layers));
    SHARED_SPLIT(sgd_kernel);
    sgd_kernel<<<dim3((unsigned)bx, a.n_layers), 256, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_ps_average(const PsAvgLayer* tab, int n_layers, long long total, int nrep, int c_bf16,
                              cudaStream_t s) {
    if (total <= 0) return cudaSuccess;
    SHARED_SPLIT(ps_average_kernel);
    ps_average_kernel<<<grid_for(total, 256), 256, 0, s>>>(tab, n_layers, total, nrep, c_bf16);
    return cudaGetLastError();
}

cudaError_t launch_mark_dropped(float* loss, float* loss_host, cudaStream_t s) {
    SHARED_SPLIT(mark_dropped_kernel);
    mark_dropped_kernel<<<1, 1, 0, s>>>(loss, loss_host);
    return cudaGetLastError();
}

cudaError_t launch_write_header(ChannelHeader* h, long long k, int batch, int version, cudaStream_t s) {
    SHARED_SPLIT(write_header_kernel);
    write_header_kernel<<<1, 1, 0, s>>>(h, k, batch, version);
    return cudaGetLastError();
}

cudaError_t launch_check_header(const ChannelHeader* h, long long k, int* status, cudaStream_t s) {
    SHARED_SPLIT(check_header_kernel);
    check_header_kernel<<<1, 1, 0, s>>>(h, k, status);
    return cudaGetLastError();
}

cudaError_t launch_wait_header(const ChannelHeader* h, long long k, long long max_iters, int* status, cudaStream_t s) {
    SHARED_SPLIT(wait_header_kernel);
    wait_header_kernel<<<1, 1, 0, s>>>(h, k, max_iters, status);
    return cudaGetLastError();
}

cudaError_t launch_cast_rows(const float* src, int rows, int d, void* dst, long long ld, int bf16, cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    SHARED_SPLIT(cast_rows_kernel);
    cast_rows_kernel<<<grid_for((long long)rows * ld, 256), 256, 0, s>>>(src, rows, d, dst, ld, bf16);
    return cudaGetLastError();
}

cudaError_t launch_stage_rows(const float* hxp, int dp, const float* hxa, int da, const int* hy, int rows, void* xp,
                              long long ld_p, void* xa, long long ld_a, int* y, int bf16, cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    const long long n = (long long)rows * (ld_p + ld_a + 1);
    SHARED_SPLIT(stage_rows_kernel);
    stage_rows_kernel<<<std::min(grid_for(n, 256), kStageBlocks), 256, 0, s>>>(hxp, dp, hxa, da, hy, rows, xp, ld_p, xa,
                                                                              ld_a, y, bf16);
    return cudaGetLastError();
}


cudaError_t launch_stage_rows_b16(const uint16_t* hxp, int dp, const uint16_t* hxa, int da, const int* hy, int rows,
                                  void* xp, long long ld_p, void* xa, long long ld_a, int* y, cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    const long long n = (long long)rows * (ld_p + ld_a + 16) / 8;
    SHARED_SPLIT(stage_rows_b16_kernel);
    stage_rows_b16_kernel<<<std::min(grid_for(n, 256), kStageBlocks), 256, 0, s>>>(hxp, dp, hxa, da, hy, rows, static_cast<uint16_t*>(xp), ld_p,
                                                          static_cast<uint16_t*>(xa), ld_a, y);
    return cudaGetLastError();
}

cudaError_t launch_to_f32(const void* src, long long ld, int rows, int cols, int bf16, float* dst, cudaStream_t s) {
    if (rows <= 0 || cols <= 0) return cudaSuccess;
    SHARED_SPLIT(to_f32_kernel);
    to_f32_kernel<<<grid_for((long long)rows * cols, 256), 256, 0, s>>>(src, ld, rows, cols, bf16, dst);
    return cudaGetLastError();
}

}  // namespace vfl
