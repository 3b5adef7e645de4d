// tcgen05 GEMMs for the bf16 Linear layers of the split-VFL step.
//
// One CTA computes one 128 x 128 fp32 accumulator tile in tensor memory:
//   warp 0     TMA producer: 128B-swizzled bf16 tiles of A and B into a
//              4-stage shared-memory ring (mbarrier full/empty pairs)
//   warp 1     allocates TMEM and issues tcgen05.mma (M=128, N=128, K=16) from
//              one thread; tcgen05.commit frees each stage and finally
//              signals the epilogue
//   warps 2-5  epilogue: tcgen05.ld of their 32-lane quarter, fused
//              bias+ReLU (forward), ReLU-mask + column split (input gradient)
//              or fp32 split-K partial store (weight gradient)
// Operands are K-major (k contiguous) or MN-major (m / n contiguous); the
// shared-memory descriptors describe both, so no transposed copies are needed:
//   FWD  C[rows, out] = X[rows, in] . W[out, in]^T     A K-major,  B K-major
//   DX   C[rows, in]  = D[rows, out] . W[out, in]      A K-major,  B MN-major
//   DW   P[out, in]   = D[rows, out]^T . X[rows, in]   A MN-major, B MN-major
// Every wait is bounded: on timeout the CTA records an error bit, drains what
// it issued (again bounded), frees its TMEM and returns.  The kernel starts with
// pdl_entry() (a captured graph may launch it programmatically) and thread 0 of
// CTA 0 checks / publishes a channel header when the step asks it to.
#include <cuda.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "vfl_tc.cuh"
#include "vfl_pdl.cuh"

namespace vfl {

namespace {

constexpr int BM = 128, BN = 128, BK = 64, STAGES = 4;
constexpr int THREADS = 192;
constexpr uint32_t TILE_BYTES = BM * BK * 2;              // 16 KB per operand per stage
constexpr uint32_t BOX_BYTES = 64 * 64 * 2;               // one MN-major box (64 mn x 64 k)
constexpr size_t SMEM_BYTES = 1024 + 2 * STAGES * TILE_BYTES + 256;
constexpr uint32_t TMEM_COLS = 128;
constexpr long long WAIT_LIMIT = 1ll << 26;               // polls before a wait is declared hung

struct TcParams {
    int mode;
    int M, N, K;
    int a_mn, b_mn;          // 1: operand is MN-major in global memory
    int ka;                  // FWD: K index where A switches to the second map
    int kb;                  // DW: N index where B switches to the second map
    int kchunk;              // DW: K range per split
    const float* bias;
    int relu;
    void* C;
    long long ldc;
    int c_f32;
    const void* mask1;
    int n_split;
    void* C2;
    long long ldc2;
    int c2_f32;
    const void* mask2;
    float* P;
    long long p_stride;
    int* err;
    HeaderOps hdr;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait on an mbarrier phase; false (and the abort flag set) on timeout.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
    for (long long it = 0; it < WAIT_LIMIT; ++it) {
        if (mbar_try(bar, parity)) return true;
        if (*abort_flag) return false;
    }
    *abort_flag = 1;
    return false;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// tcgen05 shared-memory matrix descriptor, 128-byte swizzle.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo_bytes, uint32_t sbo_bytes) {
    uint64_t d = 0;
    d |= (uint64_t)((addr & 0x3FFFF) >> 4);
    d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFF) << 16;
    d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFF) << 32;
    d |= (uint64_t)1 << 46;   // descriptor version
    d |= (uint64_t)2 << 61;   // SWIZZLE_128B
    return d;
}

// Instruction descriptor of kind::f16: bf16 A and B, fp32 D, M = 128, N = 128.
__device__ __forceinline__ uint32_t instr_desc(int a_mn, int b_mn) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)a_mn << 15) | ((uint32_t)b_mn << 16) |
           ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// bf16 bit pattern h (low 16 bits) is > 0: positive, non-zero, not NaN
__device__ __forceinline__ bool bf16_positive(uint32_t h) {
    return !(h & 0x8000u) && (h & 0x7FFFu) != 0 && (h & 0x7FFFu) <= 0x7F80u;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ float bf16_at(const void* base, long long idx) {
    return __bfloat162float(static_cast<const __nv_bfloat16*>(base)[idx]);
}

__global__ void __launch_bounds__(THREADS, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap ta2,
                   const __grid_constant__ CUtensorMap tb, const __grid_constant__ CUtensorMap tb2, const TcParams p) {
    pdl_entry();
    header_check(p.hdr);
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * TILE_BYTES;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + 2 * STAGES * TILE_BYTES);
    // bars[0..S) full, [S..2S) empty, [2S] accumulator ready, [2S+1] drain
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 2);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * BM, n0 = blockIdx.y * BN;
    int kbeg = 0, kend = p.K;
    if (p.mode == GEMM_DW) {
        kbeg = blockIdx.z * p.kchunk;
        kend = min(p.K, kbeg + p.kchunk);
    }
    const int nk = kend > kbeg ? (kend - kbeg + BK - 1) / BK : 0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(&bars[s]), 1);
            mbar_init(smem_u32(&bars[STAGES + s]), 1);
        }
        mbar_init(smem_u32(&bars[2 * STAGES]), 1);
        mbar_init(smem_u32(&bars[2 * STAGES + 1]), 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0 && nk > 0) {
        // ---------------- TMA producer ----------------
        // B tiles of a DW tile that lies past the concat split come from the second map
        const CUtensorMap* mb = &tb;
        int nb0 = n0;
        if (p.mode == GEMM_DW && n0 >= p.kb) {
            mb = &tb2;
            nb0 = n0 - p.kb;
        }
        int issued = 0;
        for (int kt = 0; kt < nk; ++kt) {
            const int s = kt % STAGES;
            const uint32_t it = kt / STAGES;
            if (!mbar_wait(smem_u32(&bars[STAGES + s]), (it & 1) ^ 1, abort_flag)) break;
            const uint32_t full = smem_u32(&bars[s]);
            mbar_expect_tx(full, 2 * TILE_BYTES);
            const int k = kbeg + kt * BK;
            const uint32_t dA = smem_u32(sA + s * TILE_BYTES), dB = smem_u32(sB + s * TILE_BYTES);
            if (!p.a_mn) {
                if (k < p.ka)
                    tma_load_2d(dA, &ta, k, m0, full);
                else
                    tma_load_2d(dA, &ta2, k - p.ka, m0, full);
            } else {
                tma_load_2d(dA, &ta, m0, k, full);
                tma_load_2d(dA + BOX_BYTES, &ta, m0 + 64, k, full);
            }
            if (!p.b_mn) {
                tma_load_2d(dB, mb, k, nb0, full);
            } else {
                tma_load_2d(dB, mb, nb0, k, full);
                tma_load_2d(dB + BOX_BYTES, mb, nb0 + 64, k, full);
            }
            issued = kt + 1;
        }
        // on abort, wait (bounded) for the loads already issued before the CTA exits
        if (*abort_flag) {
            for (int kt = (issued > STAGES ? issued - STAGES : 0); kt < issued; ++kt) {
                const uint32_t bar = smem_u32(&bars[kt % STAGES]);
                for (long long t = 0; t < WAIT_LIMIT && !mbar_try(bar, (kt / STAGES) & 1); ++t) {
                }
            }
        }
    } else if (warp == 1 && lane == 0 && nk > 0) {
        // ---------------- MMA issuer ----------------
        const uint32_t idesc = instr_desc(p.a_mn, p.b_mn);
        bool ok = true;
        for (int kt = 0; kt < nk && ok; ++kt) {
            const int s = kt % STAGES;
            if (!mbar_wait(smem_u32(&bars[s]), (kt / STAGES) & 1, abort_flag)) {
                ok = false;
                break;
            }
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t aB = smem_u32(sA + s * TILE_BYTES), bB = smem_u32(sB + s * TILE_BYTES);
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
                // K-major: the 16-element slice starts 32 bytes further along each 128-byte row;
                // MN-major: it starts 16 rows (2048 bytes) further down the 64-row box.
                const uint64_t ad = p.a_mn ? smem_desc(aB + kk * 2048, BOX_BYTES, 1024) : smem_desc(aB + kk * 32, 16, 1024);
                const uint64_t bd = p.b_mn ? smem_desc(bB + kk * 2048, BOX_BYTES, 1024) : smem_desc(bB + kk * 32, 16, 1024);
                mma_bf16(tmem, ad, bd, idesc, (kt > 0 || kk > 0) ? 1u : 0u);
            }
            mma_commit(smem_u32(&bars[STAGES + s]));
        }
        // signal the epilogue (also after an abort, so that in-flight MMAs finish before TMEM is freed)
        mma_commit(smem_u32(&bars[2 * STAGES]));
    } else if (warp >= 2) {
        // ---------------- epilogue ----------------
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const int m = m0 + row;
        bool have = nk > 0;
        if (have) {
            have = mbar_wait(smem_u32(&bars[2 * STAGES]), 0, abort_flag);
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        }
        for (int c0 = 0; c0 < BN; c0 += 32) {
            float v[32];
            if (have) {
                tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)c0, v);
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) v[i] = 0.f;
            }
            if (*abort_flag || m >= p.M) continue;
            const int nbase = n0 + c0;
            if (p.mode == GEMM_FWD) {
                __nv_bfloat16* C = static_cast<__nv_bfloat16*>(p.C) + (long long)m * p.ldc + nbase;
                if (nbase + 32 <= p.N) {
                    const float4* b4 = reinterpret_cast<const float4*>(p.bias + nbase);
                    uint32_t packed[16];
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        const float4 bq = b4[q];
                        float x0 = v[4 * q] + bq.x, x1 = v[4 * q + 1] + bq.y, x2 = v[4 * q + 2] + bq.z,
                              x3 = v[4 * q + 3] + bq.w;
                        if (p.relu) {
                            x0 = fmaxf(x0, 0.f); x1 = fmaxf(x1, 0.f); x2 = fmaxf(x2, 0.f); x3 = fmaxf(x3, 0.f);
                        }
                        packed[2 * q] = pack_bf16(x0, x1);
                        packed[2 * q + 1] = pack_bf16(x2, x3);
                    }
                    uint4* dst = reinterpret_cast<uint4*>(C);
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        dst[q] = make_uint4(packed[4 * q], packed[4 * q + 1], packed[4 * q + 2], packed[4 * q + 3]);
                } else {
                    for (int i = 0; i < 32 && nbase + i < p.N; ++i) {
                        float x = v[i] + p.bias[nbase + i];
                        if (p.relu) x = fmaxf(x, 0.f);
                        C[i] = __float2bfloat16_rn(x);
                    }
                }
            } else if (p.mode == GEMM_DX) {
                const bool to_c = nbase + 32 <= min(p.N, p.n_split);
                const bool to_c2 = nbase >= p.n_split && nbase + 32 <= p.N && ((nbase - p.n_split) & 7) == 0;
                if (to_c || to_c2) {
                    const long long idx = to_c ? (long long)m * p.ldc + nbase : (long long)m * p.ldc2 + (nbase - p.n_split);
                    const void* mask = to_c ? p.mask1 : p.mask2;
                    if (mask) {
                        const uint4* mk = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(mask) + idx);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const uint4 w = mk[q];
                            const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                            for (int h = 0; h < 4; ++h) {
                                if (!bf16_positive(ws[h] & 0xFFFFu)) v[8 * q + 2 * h] = 0.f;
                                if (!bf16_positive(ws[h] >> 16)) v[8 * q + 2 * h + 1] = 0.f;
                            }
                        }
                    }
                    if (to_c2 && p.c2_f32) {
                        float4* dst = reinterpret_cast<float4*>(static_cast<float*>(p.C2) + idx);
#pragma unroll
                        for (int q = 0; q < 8; ++q) dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                    } else {
                        uint4* dst = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(to_c ? p.C : p.C2) + idx);
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            dst[q] = make_uint4(pack_bf16(v[8 * q], v[8 * q + 1]), pack_bf16(v[8 * q + 2], v[8 * q + 3]),
                                                pack_bf16(v[8 * q + 4], v[8 * q + 5]), pack_bf16(v[8 * q + 6], v[8 * q + 7]));
                    }
                } else {
                    for (int i = 0; i < 32; ++i) {
                        const int n = nbase + i;
                        if (n >= p.N) break;
                        float x = v[i];
                        if (n < p.n_split) {
                            const long long idx = (long long)m * p.ldc + n;
                            if (p.mask1 && !(bf16_at(p.mask1, idx) > 0.f)) x = 0.f;
                            static_cast<__nv_bfloat16*>(p.C)[idx] = __float2bfloat16_rn(x);
                        } else {
                            const long long idx = (long long)m * p.ldc2 + (n - p.n_split);
                            if (p.mask2 && !(bf16_at(p.mask2, idx) > 0.f)) x = 0.f;
                            if (p.c2_f32)
                                static_cast<float*>(p.C2)[idx] = x;
                            else
                                static_cast<__nv_bfloat16*>(p.C2)[idx] = __float2bfloat16_rn(x);
                        }
                    }
                }
            } else {
                float* P = p.P + (long long)blockIdx.z * p.p_stride + (long long)m * p.ldc + nbase;
                if (nbase + 32 <= p.N && (p.ldc & 3) == 0) {
                    float4* dst = reinterpret_cast<float4*>(P);
#pragma unroll
                    for (int q = 0; q < 8; ++q) dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                } else {
                    for (int i = 0; i < 32 && nbase + i < p.N; ++i) P[i] = v[i];
                }
            }
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) atomicOr(p.err, ST_KERNEL_TIMEOUT);
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
    }
    header_publish(p.hdr);
}

// ---------------------------------------------------------------------------
// host side: tensor maps through the driver entry point
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(f);
    });
    return fn;
}

// 2-D bf16 map: `inner` contiguous elements per row, `rows` rows of `ld` elements; box inner x box_rows.
bool make_map(CUtensorMap* m, const void* base, long long inner, long long rows, long long ld, int box_inner,
              int box_rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn || !base || inner < 1 || rows < 1) return false;
    cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)box_inner, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool tc_available() { return encode_fn() != nullptr; }

bool tc_supported_fwd(int in, int out, bool concat, int ka, bool out_f32) {
    if (out_f32 || in < 1 || out < 16) return false;
    if (concat && ka % BK != 0) return false;
    return tc_available();
}

bool tc_supported_dx(int in, int out, int n_split, bool c2_f32) {
    (void)n_split;
    (void)c2_f32;
    if (in < 16 || out < 16) return false;
    return tc_available();
}

bool tc_shape_dw(int out, int in, bool concat, int kb) {
    if (out < 16 || in < 1) return false;
    return !(concat && kb % BN != 0);
}

bool tc_supported_dw(int out, int in, bool concat, int kb) { return tc_shape_dw(out, in, concat, kb) && tc_available(); }

void tc_choose_split(int out, int in, int rows, int* nsplit, int* kchunk) {
    const long long tiles = (long long)((out + BM - 1) / BM) * ((in + BN - 1) / BN);
    long long ns = std::max<long long>(1, (152 + tiles / 2) / std::max<long long>(1, tiles));
    ns = std::min<long long>(ns, std::max(1, rows / 256));
    ns = std::min<long long>(ns, 16);
    int kc = (int)(((rows + ns - 1) / ns + BK - 1) / BK * BK);
    *kchunk = kc;
    *nsplit = (rows + kc - 1) / kc;
}

cudaError_t launch_tc_gemm(const TcGemm& g, cudaStream_t s) {
    static cudaError_t attr = cudaFuncSetAttribute(tc_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   (int)SMEM_BYTES);
    if (attr != cudaSuccess) return attr;
    if (g.M <= 0 || g.N <= 0) return cudaSuccess;
    TcParams p;
    std::memset(&p, 0, sizeof p);
    p.mode = g.mode;
    p.M = g.M;
    p.N = g.N;
    p.K = g.K;
    p.err = g.err;
    p.hdr = g.hdr;
    CUtensorMap ta, ta2, tb, tb2;
    std::memset(&ta, 0, sizeof ta);
    std::memset(&ta2, 0, sizeof ta2);
    std::memset(&tb, 0, sizeof tb);
    std::memset(&tb2, 0, sizeof tb2);
    bool ok = true;
    dim3 grid((g.M + BM - 1) / BM, (g.N + BN - 1) / BN, 1);
    if (g.mode == GEMM_FWD) {
        // A = X [rows, K] (two maps when concatenated along K), B = W [out, K]
        p.a_mn = 0;
        p.b_mn = 0;
        p.ka = g.A2 ? g.ka : (1 << 30);
        const long long k1 = g.A2 ? g.ka : g.lda;
        ok &= make_map(&ta, g.A, k1, g.M, g.lda, 64, BM);
        ta2 = ta;
        if (g.A2) ok &= make_map(&ta2, g.A2, g.lda2, g.M, g.lda2, 64, BM);
        ok &= make_map(&tb, g.B, g.ldb, g.N, g.ldb, 64, BN);
        tb2 = tb;
        p.bias = g.bias;
        p.relu = g.relu;
        p.C = g.C;
        p.ldc = g.ldc;
    } else if (g.mode == GEMM_DX) {
        // A = D [rows, K = out], B(n, k) = W[k, n]: W [out rows, in_ld] is MN-major
        p.a_mn = 0;
        p.b_mn = 1;
        p.ka = 1 << 30;
        ok &= make_map(&ta, g.A, g.lda, g.M, g.lda, 64, BM);
        ta2 = ta;
        ok &= make_map(&tb, g.B, g.ldb, g.K, g.ldb, 64, 64);
        tb2 = tb;
        p.C = g.C;
        p.ldc = g.ldc;
        p.mask1 = g.mask1;
        p.n_split = g.n_split;
        p.C2 = g.C2;
        p.ldc2 = g.ldc2;
        p.c2_f32 = g.c2_f32;
        p.mask2 = g.mask2;
    } else {
        // A(m = out, k = row) = D[row, out], B(n = in, k = row) = X[row, in]: both MN-major
        p.a_mn = 1;
        p.b_mn = 1;
        p.ka = 1 << 30;
        p.kb = g.B2 ? g.kb : (1 << 30);
        ok &= make_map(&ta, g.A, g.lda, g.K, g.lda, 64, 64);
        ta2 = ta;
        const long long n1 = g.B2 ? g.kb : g.ldb;
        ok &= make_map(&tb, g.B, n1, g.K, g.ldb, 64, 64);
        tb2 = tb;
        if (g.B2) ok &= make_map(&tb2, g.B2, g.ldb2, g.K, g.ldb2, 64, 64);
        p.kchunk = g.kchunk;
        p.P = g.P;
        p.p_stride = g.p_stride;
        p.ldc = g.ldc;
        grid.z = g.nsplit;
    }
    if (!ok) return cudaErrorInvalidValue;
    tc_gemm_kernel<<<grid, THREADS, SMEM_BYTES, s>>>(ta, ta2, tb, tb2, p);
    return cudaGetLastError();
}

}  // namespace vfl
