// tcgen05 GEMMs for the bf16 Linear layers of the split-VFL step.
//
// Forward and input-gradient GEMMs (tc_gemm_kernel) are persistent: the grid is
// at most one CTA per SM and each CTA walks its 128 x BN output tiles (BN = 128
// or 256, chosen per shape) in a static round-robin order.  Warp roles:
//   warp 0     TMA producer: 128B-swizzled bf16 tiles of A and B into a ring
//              of shared-memory stages (mbarrier full / empty pairs)
//   warp 1     allocates TMEM and issues tcgen05.mma (M = 128, N = BN, K = 16)
//              from one thread; tcgen05.commit frees each stage and, after a
//              tile's last k-block, marks its accumulator full
//   warps 2-17 epilogue: tcgen05.ld of their 32-lane quarter and column quarter,
//              fused bias + ReLU (forward) or ReLU-mask + column split (input
//              gradient), staged in shared memory and stored as row segments
// Two accumulators live in TMEM (2 x BN columns), so the epilogue of one tile
// runs while the MMAs of the next tile fill the other.
//
// The weight gradient (tc_dw_kernel) splits the batch rows over the CTAs of a
// thread-block cluster: every CTA accumulates its row chunk of one 128 x BN
// tile of dW = D^T X in TMEM and writes it to its slice of an L2-resident
// workspace; after a cluster barrier (release / acquire) the CTA that owns each
// 128 / cluster-size rows of the tile sums the slices in rank order
// (deterministic).  The owner writes the reduced dW and, for parties with one
// worker stream, applies the SGD step of Eq. 2 in the same epilogue (fp32
// master and the new version's bf16 copy).  The bias gradient (column sums of
// D) is taken by the epilogue warps from the A stages in shared memory while
// the MMAs run, and reduced with the tile.
//
// Operands are K-major (k contiguous) or MN-major (m / n contiguous); the
// shared-memory descriptors describe both, so no transposed copies are needed:
//   FWD  C[rows, out] = X[rows, in] . W[out, in]^T     A K-major,  B K-major
//   DX   C[rows, in]  = D[rows, out] . W[out, in]      A K-major,  B MN-major
//   DW   P[out, in]   = D[rows, out]^T . X[rows, in]   A MN-major, B MN-major
// Every wait is bounded: on timeout the CTA records an error bit, drains what
// it issued (again bounded), frees its TMEM and returns.  Thread 0 of CTA 0
// checks / publishes a channel header when the step asks it to.
#include <cuda.h>
#include <cooperative_groups.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "vfl_tc.cuh"

namespace cg = cooperative_groups;

namespace vfl {

namespace {

constexpr int BM = 128, BK = 64;                          // K-major stages: 64 k (one 128-byte row)
constexpr int EPI_WARPS = 8;                              // weight gradient: epilogue / column-sum warps
constexpr int THREADS = 64 + 32 * EPI_WARPS;             // producer, MMA issuer, epilogue
constexpr int GEMM_EPI_WARPS = 16;                        // forward / input gradient: four per TMEM lane quarter
constexpr int GEMM_THREADS = 64 + 32 * GEMM_EPI_WARPS;
constexpr int DW_KS = 128;                                // weight-gradient stages: 128 k (MN-major boxes)
constexpr long long WAIT_LIMIT = 1ll << 26;               // polls before a wait is declared hung
constexpr int MAX_CLUSTER = 16;

// A ring of STAGES shared-memory stages, each one 128 x KS bf16 tile of A and one BN x KS tile of B.
// K-major operands come as one box (KS = 64: the 128-byte swizzle row); MN-major operands as boxes of
// 64 m / n columns by KS k rows.
template <int BN, int STAGES_, int KS_ = BK>
struct Ring {
    static constexpr int STAGES = STAGES_;
    static constexpr int N = BN;
    static constexpr int KS = KS_;
    static constexpr uint32_t A_BYTES = BM * KS * 2;
    static constexpr uint32_t B_BYTES = BN * KS * 2;
    static constexpr uint32_t BOX_BYTES = 64 * KS * 2;
    static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr uint32_t RING_BYTES = STAGES * STAGE_BYTES;
    static constexpr uint32_t CTRL_BYTES = 256;   // barriers, TMEM slot, abort flag
};

// Forward / input gradient: four (256-wide) or six (128-wide) stages keep the MMAs fed with every SM busy,
// and leave room for each epilogue warp's output staging (32 rows x 64 bytes).
template <int BN>
struct GemmCfg : Ring<BN, BN == 256 ? 4 : 6> {
    using R = Ring<BN, BN == 256 ? 4 : 6>;
    static constexpr uint32_t WARP_BYTES = 2048;
    static constexpr size_t SMEM = 1024 + R::RING_BYTES + R::CTRL_BYTES + GEMM_EPI_WARPS * WARP_BYTES;
};

// Weight gradient: 128-wide tiles, stages of 128 k rows (two MN-major boxes per operand: a stage's TMA
// work covers two 64-row k-blocks), three stages; after the mainloop the ring holds the fp32
// accumulator tile.  Column-sum scratch: 16 x 128 partials, 128 sums.
struct DwCfg : Ring<128, 3, DW_KS> {
    using R = Ring<128, 3, DW_KS>;
    static constexpr uint32_t CSUM_BYTES = (16 * 128 + 128) * 4;
    static constexpr size_t SMEM = 1024 + R::RING_BYTES + R::CTRL_BYTES + CSUM_BYTES;
    static_assert((size_t)128 * (128 + 4) * 4 <= R::RING_BYTES, "the accumulator tile must fit the ring");
};

struct TcParams {
    int mode;
    int M, N, K;
    int tiles_m, tiles_n;
    int a_mn, b_mn;
    int ka;                  // FWD: K index where A switches to the second map
    int kb;                  // DW: N index where B switches to the second map
    int kchunk;              // DW: rows per cluster rank
    const float* bias;
    int relu;
    void* C;
    long long ldc;
    const void* mask1;
    int n_split;
    void* C2;
    long long ldc2;
    int c2_f32;
    const void* mask2;
    // DW outputs
    float* P;                // reduced dW [M, N] (row stride ldp), or null
    long long ldp;
    float* Pb;               // reduced db [M], or null (no bias gradient)
    float* ws;               // per-rank partial tiles [cs][tiles][128][BN] (L2-resident exchange)
    float* wsb;              // per-rank bias partials [cs][tiles_m][128]
    float* Wm;               // fused SGD: fp32 master [M, N] (row stride N), or null
    float* bm;               //            fp32 bias master [M]
    void* cW;                //            new version's bf16 copy [M, cw_ld]
    long long cw_ld;
    float* cb;               //            new version's bias copy [M]
    float lr;
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

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
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

// The same for a wait that spans a whole mainloop (epilogue warps waiting for a tile's MMAs): a short
// sleep between polls leaves the issue slots and the shared-memory pipe to the producer and the MMA
// issuer.  Bounded like mbar_wait (about a second of sleeping).
__device__ __forceinline__ bool mbar_wait_idle(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
    for (long long it = 0; it < (WAIT_LIMIT >> 3); ++it) {
        if (mbar_try(bar, parity)) return true;
        if (*abort_flag) return false;
        __nanosleep(128);
    }
    *abort_flag = 1;
    return false;
}

// Bring a tensor map (a __grid_constant__ kernel parameter) into the TMA unit's descriptor cache ahead of
// its first copy.
__device__ __forceinline__ void prefetch_map(const CUtensorMap* map) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
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

// Instruction descriptor of kind::f16: bf16 A and B, fp32 D, M = 128, N = BN.
template <int BN>
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

// Per 16-bit half of a bf16x2 word: 0xFFFF where that bf16 is > 0 (non-zero magnitude, sign clear, not
// NaN), else 0 -- bf16_positive for both halves at once, without branches.  Magnitudes are at most
// 0x7FFF, so neither addition carries out of its half.
__device__ __forceinline__ uint32_t bf16x2_positive_mask(uint32_t w) {
    const uint32_t m = w & 0x7FFF7FFFu;
    const uint32_t nonzero = (m + 0x7FFF7FFFu) & 0x80008000u;
    const uint32_t nan = (m + 0x007F007Fu) & 0x80008000u;
    const uint32_t keep = nonzero & ~nan & ~w & 0x80008000u;
    return (keep >> 15) * 0xFFFFu;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ float bf16_at(const void* base, long long idx) {
    return __bfloat162float(static_cast<const __nv_bfloat16*>(base)[idx]);
}

// ---------------------------------------------------------------------------
// Producer: the k-blocks [kb0, kb0 + nk) of one tile into the ring, continuing
// the ring position `it` (one count per k-block over the CTA's whole run).
// ---------------------------------------------------------------------------
template <typename C>
__device__ __forceinline__ bool produce_tile(const TcParams& p, const CUtensorMap* ta, const CUtensorMap* ta2,
                                             const CUtensorMap* mb, int nb0, int m0, int kbeg, int nk, uint8_t* ring,
                                             uint64_t* full, uint64_t* empty, uint32_t& it, volatile int* abort_flag) {
    constexpr int BN = C::N;
    for (int kt = 0; kt < nk; ++kt, ++it) {
        const int s = it % C::STAGES;
        if (!mbar_wait(smem_u32(&empty[s]), ((it / C::STAGES) & 1) ^ 1, abort_flag)) return false;
        const uint32_t bar = smem_u32(&full[s]);
        mbar_expect_tx(bar, C::STAGE_BYTES);
        const int k = kbeg + kt * C::KS;
        const uint32_t dA = smem_u32(ring + s * C::STAGE_BYTES), dB = dA + C::A_BYTES;
        if (!p.a_mn) {
            if (k < p.ka)
                tma_load_2d(dA, ta, k, m0, bar);
            else
                tma_load_2d(dA, ta2, k - p.ka, m0, bar);
        } else {
            tma_load_2d(dA, ta, m0, k, bar);
            tma_load_2d(dA + C::BOX_BYTES, ta, m0 + 64, k, bar);
        }
        if (!p.b_mn) {
            tma_load_2d(dB, mb, k, nb0, bar);
        } else {
#pragma unroll
            for (int j = 0; j < BN / 64; ++j) tma_load_2d(dB + j * C::BOX_BYTES, mb, nb0 + 64 * j, k, bar);
        }
    }
    return true;
}

// After an abort: wait (bounded) for the loads of the last STAGES ring positions before the CTA exits.
template <typename C>
__device__ __forceinline__ void drain_loads(uint64_t* full, uint32_t issued) {
    const uint32_t first = issued > (uint32_t)C::STAGES ? issued - C::STAGES : 0;
    for (uint32_t i = first; i < issued; ++i) {
        const uint32_t bar = smem_u32(&full[i % C::STAGES]);
        for (long long t = 0; t < WAIT_LIMIT && !mbar_try(bar, (i / C::STAGES) & 1); ++t) {
        }
    }
}

// MMA issue for one tile's k-blocks into accumulator `acc`.
template <typename C>
__device__ __forceinline__ bool mma_tile(const TcParams& p, uint32_t acc, int nk, uint8_t* ring, uint64_t* full,
                                         uint64_t* empty, uint32_t& it, volatile int* abort_flag) {
    const uint32_t idesc = instr_desc<C::N>(p.a_mn, p.b_mn);
    for (int kt = 0; kt < nk; ++kt, ++it) {
        const int s = it % C::STAGES;
        if (!mbar_wait(smem_u32(&full[s]), (it / C::STAGES) & 1, abort_flag)) return false;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t aB = smem_u32(ring + s * C::STAGE_BYTES), bB = aB + C::A_BYTES;
#pragma unroll
        for (int kk = 0; kk < C::KS / 16; ++kk) {
            // K-major: the 16-element slice starts 32 bytes further along each 128-byte row;
            // MN-major: it starts 16 rows (2048 bytes) further down each box of KS rows.
            const uint64_t ad =
                p.a_mn ? smem_desc(aB + kk * 2048, C::BOX_BYTES, 1024) : smem_desc(aB + kk * 32, 16, 1024);
            const uint64_t bd =
                p.b_mn ? smem_desc(bB + kk * 2048, C::BOX_BYTES, 1024) : smem_desc(bB + kk * 32, 16, 1024);
            mma_bf16(acc, ad, bd, idesc, (kt > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(smem_u32(&empty[s]));
    }
    return true;
}

// Input-gradient epilogue of one 32-column chunk for row m, one row per lane: the passes that straddle
// the split column between C and C2.
__device__ __forceinline__ void epilogue_chunk(const TcParams& p, int m, int nbase, float* v) {
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
}

// ---------------------------------------------------------------------------
// Staged epilogue.  A warp owns 32 accumulator rows (its TMEM lane quarter); per pass it takes 32 columns
// (16 for fp32 output), writes them row per lane into its 32 x 64-byte staging buffer, then reads them
// back so that four lanes cover one row's 64 bytes and stores whole row segments: every store
// instruction writes eight full 64-byte pieces of rows.  Two rows share a 128-byte line; the line's
// eight 16-byte units are XOR-swizzled by the line index, so both directions are conflict-free.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t stage_unit(uint32_t stage, int r, int ch) {
    const int line = r >> 1;
    const int unit = (((r & 1) << 2) | ch) ^ (line & 7);
    return stage + (uint32_t)(line * 128 + unit * 16);
}
__device__ __forceinline__ void sts128(uint32_t a, uint4 v) {
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w) : "memory");
}
__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a) : "memory");
    return v;
}

// The bf16 ReLU mask an input-gradient pass of 32 columns from nb applies, with its row stride and first
// column (masks share the layout of the matrix they gate); null for forward, fp32-output or straddling passes.
__device__ __forceinline__ const __nv_bfloat16* dx_pass_mask(const TcParams& p, int nb, long long* ld, int* n) {
    if (p.mode == GEMM_FWD || nb >= p.N) return nullptr;
    const int cols = min(32, p.N - nb);
    if (nb + cols <= p.n_split) {
        *ld = p.ldc;
        *n = nb;
        return static_cast<const __nv_bfloat16*>(p.mask1);
    }
    if (nb >= p.n_split && ((nb - p.n_split) & 7) == 0 && !p.c2_f32) {
        *ld = p.ldc2;
        *n = nb - p.n_split;
        return static_cast<const __nv_bfloat16*>(p.mask2);
    }
    return nullptr;
}

// This lane's four 8-column mask units of a 32 x 32 block (the units store_bf16_block writes), read
// ahead of the stores so that their latency overlaps the accumulator wait or the previous pass.
__device__ __forceinline__ void load_mask_block(const __nv_bfloat16* mask, long long ld, int lane, int r0, int rows,
                                                int n, int cols, uint4 (&mk)[4]) {
    const int c = (lane & 3) * 8;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int r = i * 8 + (lane >> 2);
        mk[i] = make_uint4(0u, 0u, 0u, 0u);
        if (mask && r0 + r < rows && c + 8 <= cols)
            mk[i] = __ldg(reinterpret_cast<const uint4*>(mask + (long long)(r0 + r) * ld + n + c));
    }
}

// Read back the staged 32 x 32 bf16 block and store rows [r0, r0 + 32) x columns [n, n + 32) of a bf16
// matrix (row stride ld, `cols` valid columns from n), masked by mask > 0 when mask is set: full 8-column
// units take the mask from mk (load_mask_block), a ragged last unit reads it element by element.
__device__ __forceinline__ void store_bf16_block(uint32_t stage, int lane, __nv_bfloat16* C, long long ld,
                                                 const __nv_bfloat16* mask, const uint4 (&mk)[4], int r0, int rows,
                                                 int n, int cols) {
    const int ch = lane & 3;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int r = i * 8 + (lane >> 2);
        if (r0 + r >= rows) continue;
        uint4 d = lds128(stage_unit(stage, r, ch));
        const int c = ch * 8;
        const long long idx = (long long)(r0 + r) * ld + n + c;
        if (c + 8 <= cols) {
            if (mask) {
                d.x &= bf16x2_positive_mask(mk[i].x);
                d.y &= bf16x2_positive_mask(mk[i].y);
                d.z &= bf16x2_positive_mask(mk[i].z);
                d.w &= bf16x2_positive_mask(mk[i].w);
            }
            *reinterpret_cast<uint4*>(C + idx) = d;
        } else {
            const __nv_bfloat16* h = reinterpret_cast<const __nv_bfloat16*>(&d);
            for (int e = 0; e < 8 && c + e < cols; ++e) {
                __nv_bfloat16 x = h[e];
                if (mask && !(__bfloat162float(mask[idx + e]) > 0.f)) x = __float2bfloat16_rn(0.f);
                C[idx + e] = x;
            }
        }
    }
}

// The same for 16 fp32 columns per pass (64 bytes a row): v[16] of row `lane` into the staging buffer,
// then rows [r0, r0 + 32) x columns [n, n + 16) of an fp32 matrix, masked by a bf16 mask when set.
__device__ __forceinline__ void store_f32_block(uint32_t stage, int lane, const float* v, float* C, long long ld,
                                                const __nv_bfloat16* mask, int r0, int rows, int n, int cols) {
#pragma unroll
    for (int c = 0; c < 4; ++c)
        sts128(stage_unit(stage, lane, c), make_uint4(__float_as_uint(v[4 * c]), __float_as_uint(v[4 * c + 1]),
                                                      __float_as_uint(v[4 * c + 2]), __float_as_uint(v[4 * c + 3])));
    __syncwarp();
    const int ch = lane & 3;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int r = i * 8 + (lane >> 2);
        if (r0 + r >= rows) continue;
        const uint4 du = lds128(stage_unit(stage, r, ch));
        const float4 d = make_float4(__uint_as_float(du.x), __uint_as_float(du.y), __uint_as_float(du.z), __uint_as_float(du.w));
        const int c = ch * 4;
        const long long idx = (long long)(r0 + r) * ld + n + c;
        float dv[4] = {d.x, d.y, d.z, d.w};
        for (int e = 0; e < 4; ++e)
            if (mask && c + e < cols && !(__bfloat162float(mask[idx + e]) > 0.f)) dv[e] = 0.f;
        if (c + 4 <= cols)
            *reinterpret_cast<float4*>(C + idx) = make_float4(dv[0], dv[1], dv[2], dv[3]);
        else
            for (int e = 0; e < 4 && c + e < cols; ++e) C[idx + e] = dv[e];
    }
    __syncwarp();
}

// ---------------------------------------------------------------------------
// Persistent forward / input-gradient GEMM.
// ---------------------------------------------------------------------------
template <int BN>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap ta2,
                   const __grid_constant__ CUtensorMap tb, const TcParams p) {
    using C = GemmCfg<BN>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(ring + C::RING_BYTES);
    uint64_t* empty = full + C::STAGES;
    uint64_t* acc_full = empty + C::STAGES;      // [2]
    uint64_t* acc_empty = acc_full + 2;          // [2]
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ntiles = p.tiles_m * p.tiles_n;
    const int nk = (p.K + BK - 1) / BK;

    if (threadIdx.x == 32) {
        prefetch_map(&ta);
        prefetch_map(&ta2);
        prefetch_map(&tb);
    }
    if (threadIdx.x == 0) {
        for (int s = 0; s < C::STAGES; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&acc_full[b]), 1);
            mbar_init(smem_u32(&acc_empty[b]), GEMM_EPI_WARPS);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(2 * BN)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_slot;
    // set-up above overlaps the previous kernel's tail (this CTA's shared memory and TMEM are its own:
    // no other tensor-core CTA fits the SM beside it); inputs are read only after that kernel completes
    asm volatile("griddepcontrol.wait;" ::: "memory");
    header_check(p.hdr);

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer ----------------
        uint32_t it = 0;
        for (int t = blockIdx.x; t < ntiles && nk > 0; t += gridDim.x) {
            const int m0 = (t / p.tiles_n) * BM, n0 = (t % p.tiles_n) * BN;
            if (!produce_tile<C>(p, &ta, &ta2, &tb, n0, m0, 0, nk, ring, full, empty, it, abort_flag)) break;
        }
        if (*abort_flag) drain_loads<C>(full, it);
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer ----------------
        uint32_t it = 0;
        int i = 0;
        for (int t = blockIdx.x; t < ntiles && nk > 0; t += gridDim.x, ++i) {
            const int b = i & 1;
            if (!mbar_wait(smem_u32(&acc_empty[b]), ((i >> 1) & 1) ^ 1, abort_flag)) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const bool ok = mma_tile<C>(p, tmem + (uint32_t)(b * BN), nk, ring, full, empty, it, abort_flag);
            // mark the accumulator full (also after an abort, so that in-flight MMAs finish before TMEM is freed)
            mma_commit(smem_u32(&acc_full[b]));
            if (!ok) break;
        }
    } else if (warp >= 2) {
        // ---------------- epilogue ----------------
        // 16 warps: warp w reads TMEM lane quarter w mod 4 (the only lanes it may access) and one quarter
        // of the tile's columns, NP passes of 32
        constexpr int NP = BN / 128;
        const int quarter = warp & 3;
        const int group = (warp - 2) >> 2;
        const int cbeg = group * (BN / 4);
        const uint32_t stage = smem_u32(ring + C::RING_BYTES + C::CTRL_BYTES + (warp - 2) * C::WARP_BYTES);
        int i = 0;
        for (int t = blockIdx.x; t < ntiles && nk > 0; t += gridDim.x, ++i) {
            const int b = i & 1;
            const int m0 = (t / p.tiles_n) * BM, n0 = (t % p.tiles_n) * BN;
            const int r0 = m0 + quarter * 32;
            // read while the tile's MMAs run: this warp's columns' bias (lane j of pass q holds column
            // cbeg + 32 q + j) and, for the input gradient, the ReLU masks of its passes
            float bias[NP];
            uint4 mk[NP][4];
#pragma unroll
            for (int q = 0; q < NP; ++q) {
                const int nq = n0 + cbeg + 32 * q;
                bias[q] = p.mode == GEMM_FWD && nq + lane < p.N ? __ldg(p.bias + nq + lane) : 0.f;
                long long mld = 0;
                int mn = 0;
                const __nv_bfloat16* mp = dx_pass_mask(p, nq, &mld, &mn);
                load_mask_block(mp, mld, lane, r0, p.M, mn, min(32, p.N - nq), mk[q]);
            }
            if (!mbar_wait_idle(smem_u32(&acc_full[b]), (i >> 1) & 1, abort_flag)) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
            for (int q = 0; q < NP; ++q) {
                const int c0 = cbeg + 32 * q;
                float v[32];
                tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(b * BN + c0), v);
                const int nb = n0 + c0;
                if (__any_sync(0xffffffffu, *abort_flag != 0) || nb >= p.N) continue;
                const int cols = min(32, p.N - nb);
                if (p.mode == GEMM_FWD) {
                    uint32_t u[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        float x0 = v[2 * j] + __shfl_sync(0xffffffffu, bias[q], 2 * j);
                        float x1 = v[2 * j + 1] + __shfl_sync(0xffffffffu, bias[q], 2 * j + 1);
                        if (p.relu) {
                            x0 = fmaxf(x0, 0.f);
                            x1 = fmaxf(x1, 0.f);
                        }
                        u[j] = pack_bf16(x0, x1);
                    }
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        sts128(stage_unit(stage, lane, c), make_uint4(u[4 * c], u[4 * c + 1], u[4 * c + 2], u[4 * c + 3]));
                    __syncwarp();
                    store_bf16_block(stage, lane, static_cast<__nv_bfloat16*>(p.C), p.ldc, nullptr, mk[q], r0, p.M,
                                     nb, cols);
                    __syncwarp();
                } else if (nb + cols <= p.n_split || (nb >= p.n_split && ((nb - p.n_split) & 7) == 0)) {
                    // the input gradient: columns < n_split to C (masked by mask1), the rest to C2
                    const bool to_c = nb < p.n_split;
                    const __nv_bfloat16* mk_ptr = static_cast<const __nv_bfloat16*>(to_c ? p.mask1 : p.mask2);
                    if (!to_c && p.c2_f32) {
                        store_f32_block(stage, lane, v, static_cast<float*>(p.C2), p.ldc2, mk_ptr, r0, p.M,
                                        nb - p.n_split, min(16, cols));
                        if (cols > 16)
                            store_f32_block(stage, lane, v + 16, static_cast<float*>(p.C2), p.ldc2, mk_ptr, r0, p.M,
                                            nb + 16 - p.n_split, cols - 16);
                    } else {
#pragma unroll
                        for (int c = 0; c < 4; ++c)
                            sts128(stage_unit(stage, lane, c),
                                   make_uint4(pack_bf16(v[8 * c], v[8 * c + 1]), pack_bf16(v[8 * c + 2], v[8 * c + 3]),
                                              pack_bf16(v[8 * c + 4], v[8 * c + 5]), pack_bf16(v[8 * c + 6], v[8 * c + 7])));
                        __syncwarp();
                        store_bf16_block(stage, lane, static_cast<__nv_bfloat16*>(to_c ? p.C : p.C2),
                                         to_c ? p.ldc : p.ldc2, mk_ptr, mk[q], r0, p.M,
                                         to_c ? nb : nb - p.n_split, cols);
                        __syncwarp();
                    }
                } else if (r0 + lane < p.M) {
                    // a pass across the split column: one row per lane
                    epilogue_chunk(p, r0 + lane, nb, v);
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&acc_empty[b]));
        }
    }
    // the next kernel of the stream may start its launch while this grid drains
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) atomicOr(p.err, ST_KERNEL_TIMEOUT);
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(2 * BN) : "memory");
    }
    header_publish(p.hdr);
}

// ---------------------------------------------------------------------------
// Weight gradient with the split-K reduction in the cluster (and the SGD).
// Grid (cluster size, tiles_n, tiles_m); cluster (cluster size, 1, 1).
// ---------------------------------------------------------------------------
constexpr int DW_BN = 128;
constexpr int DW_SLD = DW_BN + 4;   // accumulator rows in shared memory, padded (conflict-free 16-byte stores)

// Owner phase: rows [r_lo, r_lo + rpo) of the tile, four columns a thread, the CS ranks' partial tiles
// (own slice included: every rank wrote its slice before the cluster barrier) summed in rank order.  A
// thread takes its groups two at a time and issues every load of both (the CS slices and, with the SGD,
// the masters) before it stores anything.  Writes dW and, with the SGD, the master and the new version's
// bf16 copy, 16 bytes (8 for the copy) a store where the row layout allows.
template <int CS>
__device__ __forceinline__ void dw_owner(const TcParams& p, const float* __restrict__ ws, size_t zstride, int r_lo,
                                         int rpo, int m0, int n0) {
    float* __restrict__ Wm = p.Wm;
    float* __restrict__ P = p.P;
    __nv_bfloat16* __restrict__ cW = static_cast<__nv_bfloat16*>(p.cW);
    const int nq = rpo * (DW_BN / 4);
    const bool vec = (p.N & 3) == 0 && (p.ldp & 3) == 0 && (p.cw_ld & 3) == 0;
    for (int e0 = threadIdx.x; e0 < nq; e0 += 2 * THREADS) {
        float4 t[2][CS];
        float4 w[2];
        int m[2], n[2], nn[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int e = e0 + h * THREADS;
            const int r = r_lo + e / (DW_BN / 4), c = (e % (DW_BN / 4)) * 4;
            m[h] = m0 + r;
            n[h] = n0 + c;
            nn[h] = (e < nq && m[h] < p.M && n[h] < p.N) ? min(4, p.N - n[h]) : 0;
            w[h] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (nn[h] == 0) continue;
            const float4* src = reinterpret_cast<const float4*>(ws + (size_t)r * DW_BN + c);
#pragma unroll
            for (int z = 0; z < CS; ++z) t[h][z] = __ldcg(src + z * (zstride / 4));
            if (Wm) {
                const float* wp = Wm + (long long)m[h] * p.N + n[h];
                if (vec && nn[h] == 4) {
                    w[h] = *reinterpret_cast<const float4*>(wp);
                } else {
                    w[h].x = wp[0];
                    if (nn[h] > 1) w[h].y = wp[1];
                    if (nn[h] > 2) w[h].z = wp[2];
                    if (nn[h] > 3) w[h].w = wp[3];
                }
            }
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            if (nn[h] == 0) continue;
            float4 g = t[h][0];
#pragma unroll
            for (int z = 1; z < CS; ++z) {
                g.x += t[h][z].x; g.y += t[h][z].y; g.z += t[h][z].z; g.w += t[h][z].w;
            }
            const float gv[4] = {g.x, g.y, g.z, g.w};
            const float wv[4] = {w[h].x - p.lr * g.x, w[h].y - p.lr * g.y, w[h].z - p.lr * g.z, w[h].w - p.lr * g.w};
            if (vec && nn[h] == 4) {
                if (P) *reinterpret_cast<float4*>(P + (long long)m[h] * p.ldp + n[h]) = g;
                if (Wm) {
                    *reinterpret_cast<float4*>(Wm + (long long)m[h] * p.N + n[h]) =
                        make_float4(wv[0], wv[1], wv[2], wv[3]);
                    *reinterpret_cast<uint2*>(cW + (long long)m[h] * p.cw_ld + n[h]) =
                        make_uint2(pack_bf16(wv[0], wv[1]), pack_bf16(wv[2], wv[3]));
                }
            } else {
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    if (j >= nn[h]) break;
                    if (P) P[(long long)m[h] * p.ldp + n[h] + j] = gv[j];
                    if (Wm) {
                        Wm[(long long)m[h] * p.N + n[h] + j] = wv[j];
                        cW[(long long)m[h] * p.cw_ld + n[h] + j] = __float2bfloat16_rn(wv[j]);
                    }
                }
            }
        }
    }
}

// The single-rank case: the tile straight from shared memory.
__device__ __forceinline__ void dw_owner_local(const TcParams& p, const float* S, int m0, int n0) {
    for (int e = threadIdx.x; e < BM * DW_BN; e += THREADS) {
        const int r = e / DW_BN, c = e % DW_BN;
        const int m = m0 + r, n = n0 + c;
        if (m >= p.M || n >= p.N) continue;
        const float g = S[r * DW_SLD + c];
        if (p.P) p.P[(long long)m * p.ldp + n] = g;
        if (p.Wm) {
            const long long idx = (long long)m * p.N + n;
            const float wn = p.Wm[idx] - p.lr * g;
            p.Wm[idx] = wn;
            static_cast<__nv_bfloat16*>(p.cW)[(long long)m * p.cw_ld + n] = __float2bfloat16_rn(wn);
        }
    }
}

__global__ void __launch_bounds__(THREADS, 1)
    tc_dw_kernel(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
                 const __grid_constant__ CUtensorMap tb2, const TcParams p) {
    using C = DwCfg;
    constexpr int BN = DW_BN;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(ring + C::RING_BYTES);
    uint64_t* empty = full + C::STAGES;
    uint64_t* acc_full = empty + C::STAGES;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 2);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    float* csum_part = reinterpret_cast<float*>(ring + C::RING_BYTES + C::CTRL_BYTES);   // [16][128]
    float* csum = csum_part + 16 * 128;                                                    // [128]

    cg::cluster_group cluster = cg::this_cluster();
    const int cs = (int)cluster.num_blocks();
    const int rank = (int)cluster.block_rank();
    const int rpo = BM / cs;                     // tile rows each rank owns in the reduction
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.z * BM, n0 = blockIdx.y * BN;
    const int kbeg = rank * p.kchunk;
    const int kend = min(p.K, kbeg + p.kchunk);
    const int nk = kend > kbeg ? (kend - kbeg + C::KS - 1) / C::KS : 0;
    const bool bias = p.Pb != nullptr && blockIdx.y == 0;   // one column of tiles takes db

    if (threadIdx.x == 32) {
        prefetch_map(&ta);
        prefetch_map(&tb);
        prefetch_map(&tb2);
    }
    if (threadIdx.x == 0) {
        for (int s = 0; s < C::STAGES; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&empty[s]), bias ? 1 + EPI_WARPS : 1);
        }
        mbar_init(smem_u32(&acc_full[0]), 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(BN)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_slot;
    asm volatile("griddepcontrol.wait;" ::: "memory");

    if (warp == 0 && lane == 0) {
        // B tiles past the concat split come from the second map
        const CUtensorMap* mb = &tb;
        int nb0 = n0;
        if (n0 >= p.kb) {
            mb = &tb2;
            nb0 = n0 - p.kb;
        }
        uint32_t it = 0;
        if (nk > 0) produce_tile<C>(p, &ta, &ta, mb, nb0, m0, kbeg, nk, ring, full, empty, it, abort_flag);
        if (*abort_flag) drain_loads<C>(full, it);
    } else if (warp == 1 && lane == 0) {
        uint32_t it = 0;
        if (nk > 0) mma_tile<C>(p, tmem, nk, ring, full, empty, it, abort_flag);
        mma_commit(smem_u32(&acc_full[0]));
    } else if (warp >= 2 && bias) {
        // column sums of the A stages (D[rows, m] MN-major: two 64-column boxes of KS rows x 128 bytes,
        // 16-byte chunks swizzled by row mod 8): thread e takes the 8 columns of chunk e mod 16 over the
        // rows r = e / 16 + 16 i of each stage, one 16-byte load a row
        const int e = threadIdx.x - 64;
        const int cg = e & 15, rg = e >> 4;
        const int box = cg >> 3, c8 = cg & 7;
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int kt = 0; kt < nk; ++kt) {
            const int s = kt % C::STAGES;
            if (!mbar_wait(smem_u32(&full[s]), (kt / C::STAGES) & 1, abort_flag)) break;
            const uint8_t* a = ring + s * C::STAGE_BYTES + box * C::BOX_BYTES;
#pragma unroll
            for (int r = rg; r < C::KS; r += 16) {
                const uint4 w = *reinterpret_cast<const uint4*>(a + r * 128 + ((c8 ^ (r & 7)) << 4));
                const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&w);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float2 f = __bfloat1622float2(h[q]);
                    acc[2 * q] += f.x;
                    acc[2 * q + 1] += f.y;
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&empty[s]));
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) csum_part[rg * 128 + cg * 8 + q] = acc[q];
    }
    if (warp >= 2) {
        if (!mbar_wait_idle(smem_u32(&acc_full[0]), 0, abort_flag)) {
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    }
    __syncthreads();
    if (bias && threadIdx.x < BM) {
        float t = 0.f;
        for (int g = 0; g < 16; ++g) t += csum_part[g * 128 + threadIdx.x];   // row groups in order
        csum[threadIdx.x] = t;
    }

    // the accumulator tile into shared memory (the ring is free: every MMA and every load is complete),
    // one row per thread
    float* S = reinterpret_cast<float*>(ring);
    if (warp >= 2) {
        const int quarter = warp & 3, half = (warp - 2) >> 2;
        const int row = quarter * 32 + lane;
#pragma unroll 1
        for (int c0 = half * (BN / 2); c0 < (half + 1) * (BN / 2); c0 += 32) {
            float v[32];
            if (nk > 0 && !*abort_flag) {
                tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)c0, v);
            } else {
#pragma unroll
                for (int q = 0; q < 32; ++q) v[q] = 0.f;
            }
            float4* d4 = reinterpret_cast<float4*>(S + row * DW_SLD + c0);
#pragma unroll
            for (int q = 0; q < 8; ++q) d4[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();

    const int tiles = p.tiles_m * p.tiles_n;
    const int tile = blockIdx.z * p.tiles_n + blockIdx.y;
    if (cs == 1) {
        dw_owner_local(p, S, m0, n0);
    } else {
        // the tile into this rank's workspace slice (row-major 128 x BN, L2-resident, coalesced), then a
        // cluster barrier (release / acquire) before the owners read the slices
        float4* dst = reinterpret_cast<float4*>(p.ws + ((size_t)rank * tiles + tile) * BM * BN);
        for (int e = threadIdx.x; e < BM * BN / 4; e += THREADS) {
            const int r = e / (BN / 4), c = (e % (BN / 4)) * 4;
            dst[e] = *reinterpret_cast<const float4*>(S + r * DW_SLD + c);
        }
        if (bias)
            for (int r = threadIdx.x; r < BM; r += THREADS) p.wsb[((size_t)rank * p.tiles_m + blockIdx.z) * BM + r] = csum[r];
        cluster.sync();
        const size_t zstride = (size_t)tiles * BM * BN;
        const float* ws = p.ws + (size_t)tile * BM * BN;
        switch (cs) {
            case 2: dw_owner<2>(p, ws, zstride, rank * rpo, rpo, m0, n0); break;
            case 4: dw_owner<4>(p, ws, zstride, rank * rpo, rpo, m0, n0); break;
            case 8: dw_owner<8>(p, ws, zstride, rank * rpo, rpo, m0, n0); break;
            default: dw_owner<16>(p, ws, zstride, rank * rpo, rpo, m0, n0); break;
        }
    }
    if (bias && threadIdx.x < rpo) {
        const int r = rank * rpo + threadIdx.x;
        const int m = m0 + r;
        if (m < p.M) {
            double g = 0.0;       // the bias partials largely cancel: sum them in fp64
            for (int z = 0; z < cs; ++z)
                g += z == rank ? csum[r] : __ldcg(p.wsb + ((size_t)z * p.tiles_m + blockIdx.z) * BM + r);
            p.Pb[m] = (float)g;
            if (p.bm) {
                const float b = p.bm[m] - p.lr * (float)g;
                p.bm[m] = b;
                p.cb[m] = b;
            }
        }
    }
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) atomicOr(p.err, ST_KERNEL_TIMEOUT);
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(BN) : "memory");
    }
}

// ---------------------------------------------------------------------------
// Layer chain: a bottom model's forward (every layer <= 256 wide) for one 128-row tile in one CTA.
// The tile's activations stay in shared memory between layers as the next layer's A operand (K-major,
// 128-byte swizzle: the epilogue writes them in the layout TMA would), only the weights stream through
// the ring, and every layer's output also goes to global memory (the backward reads it).
// ---------------------------------------------------------------------------
constexpr int CH_MAX_LAYERS = 4;
constexpr int CH_STAGES = 4;
constexpr uint32_t CH_KB_BYTES = BM * BK * 2;          // one 128 x 64 k-block of the activation tile
constexpr uint32_t CH_ACT_BYTES = 4 * CH_KB_BYTES;     // inputs up to 256 wide
constexpr uint32_t CH_B_BYTES = 256 * BK * 2;          // one weight k-block of the widest layer
constexpr uint32_t CH_RING_OFF = CH_ACT_BYTES;
constexpr uint32_t CH_CTRL_OFF = CH_RING_OFF + CH_STAGES * CH_B_BYTES;
constexpr uint32_t CH_STAGE_OFF = CH_CTRL_OFF + 256;
constexpr size_t CH_SMEM = 1024 + CH_STAGE_OFF + GEMM_EPI_WARPS * 2048;

struct ChainParams {
    int L, M, K0;
    int out[CH_MAX_LAYERS];
    const float* bias[CH_MAX_LAYERS];
    void* Y[CH_MAX_LAYERS];
    long long ldy[CH_MAX_LAYERS];
    int* err;
    HeaderOps hdr;
};
struct ChainMaps {
    CUtensorMap x;
    CUtensorMap w[CH_MAX_LAYERS];
};

__device__ __forceinline__ uint32_t idesc_n(int n) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
}

__global__ void __launch_bounds__(GEMM_THREADS, 1)
    tc_chain_kernel(const __grid_constant__ ChainMaps maps, const __grid_constant__ ChainParams p) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* act = base;
    uint8_t* ring = base + CH_RING_OFF;
    uint64_t* full = reinterpret_cast<uint64_t*>(base + CH_CTRL_OFF);
    uint64_t* empty = full + CH_STAGES;
    uint64_t* act_full = empty + CH_STAGES;    // the first layer's input tile landed (TMA)
    uint64_t* acc_full = act_full + 1;         // a layer's MMAs are complete
    uint64_t* act_ready = acc_full + 1;        // a layer's output is in `act` and TMEM is drained
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(act_ready + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * BM;
    const int L = p.L;

    if (threadIdx.x == 32) {
        prefetch_map(&maps.x);
        for (int l = 0; l < L; ++l) prefetch_map(&maps.w[l]);
    }
    if (threadIdx.x == 0) {
        for (int s = 0; s < CH_STAGES; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        mbar_init(smem_u32(act_full), 1);
        mbar_init(smem_u32(acc_full), 1);
        mbar_init(smem_u32(act_ready), GEMM_EPI_WARPS);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    // the activation tile starts at zero (columns no layer writes are read against zero weight columns);
    // the generic-proxy writes are ordered before the tensor core's and the TMA's accesses
    for (int i = threadIdx.x; i < (int)(CH_ACT_BYTES / 16); i += GEMM_THREADS)
        sts128(smem_u32(act) + 16u * i, make_uint4(0u, 0u, 0u, 0u));
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(256)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = *tmem_slot;
    asm volatile("griddepcontrol.wait;" ::: "memory");
    header_check(p.hdr);

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer: the input tile, then every layer's weight k-blocks ----------------
        const int nk0 = (p.K0 + BK - 1) / BK;
        mbar_expect_tx(smem_u32(act_full), (uint32_t)nk0 * CH_KB_BYTES);
        for (int kb = 0; kb < nk0; ++kb)
            tma_load_2d(smem_u32(act + kb * CH_KB_BYTES), &maps.x, kb * BK, m0, smem_u32(act_full));
        uint32_t it = 0;
        bool ok = true;
        for (int l = 0; l < L && ok; ++l) {
            const int in = l == 0 ? p.K0 : p.out[l - 1];
            const int nk = (in + BK - 1) / BK;
            for (int kb = 0; kb < nk; ++kb, ++it) {
                const int s = it % CH_STAGES;
                if (!mbar_wait(smem_u32(&empty[s]), ((it / CH_STAGES) & 1) ^ 1, abort_flag)) {
                    ok = false;
                    break;
                }
                const uint32_t bar = smem_u32(&full[s]);
                mbar_expect_tx(bar, (uint32_t)p.out[l] * BK * 2);
                tma_load_2d(smem_u32(ring + s * CH_B_BYTES), &maps.w[l], kb * BK, 0, bar);
            }
        }
        if (*abort_flag) {
            // bounded drain of the loads in flight before the CTA may exit
            const uint32_t first = it > (uint32_t)CH_STAGES ? it - CH_STAGES : 0;
            for (uint32_t i = first; i < it; ++i)
                for (long long t = 0; t < WAIT_LIMIT && !mbar_try(smem_u32(&full[i % CH_STAGES]), (i / CH_STAGES) & 1); ++t) {
                }
            for (long long t = 0; t < WAIT_LIMIT && !mbar_try(smem_u32(act_full), 0); ++t) {
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer ----------------
        uint32_t it = 0;
        int commits = 0;
        for (int l = 0; l < L; ++l) {
            const bool ok = l == 0 ? mbar_wait(smem_u32(act_full), 0, abort_flag)
                                   : mbar_wait(smem_u32(act_ready), (l - 1) & 1, abort_flag);
            if (!ok) {
                mma_commit(smem_u32(acc_full));
                ++commits;
                break;
            }
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const int in = l == 0 ? p.K0 : p.out[l - 1];
            const int nk = (in + BK - 1) / BK;
            const uint32_t idesc = idesc_n(p.out[l]);
            bool good = true;
            for (int kb = 0; kb < nk; ++kb, ++it) {
                const int s = it % CH_STAGES;
                if (!mbar_wait(smem_u32(&full[s]), (it / CH_STAGES) & 1, abort_flag)) {
                    good = false;
                    break;
                }
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t aB = smem_u32(act + kb * CH_KB_BYTES), bB = smem_u32(ring + s * CH_B_BYTES);
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk)
                    mma_bf16(tmem, smem_desc(aB + kk * 32, 16, 1024), smem_desc(bB + kk * 32, 16, 1024), idesc,
                             (kb > 0 || kk > 0) ? 1u : 0u);
                mma_commit(smem_u32(&empty[s]));
            }
            mma_commit(smem_u32(acc_full));
            ++commits;
            if (!good) break;
        }
        // the last commit tracks every MMA issued: wait (bounded) for it before TMEM can be freed
        if (commits > 0)
            for (long long t = 0; t < WAIT_LIMIT && !mbar_try(smem_u32(acc_full), (commits - 1) & 1); ++t) {
            }
    } else if (warp >= 2) {
        // ---------------- epilogue: 16 warps, four per TMEM lane quarter, a quarter of the columns each ----
        const int quarter = warp & 3;
        const int group = (warp - 2) >> 2;
        const int row = quarter * 32 + lane;            // this lane's row of the tile
        const int r0 = m0 + quarter * 32;
        const uint32_t stage = smem_u32(base + CH_STAGE_OFF + (warp - 2) * 2048);
        const uint4 nomask[4] = {};
        for (int l = 0; l < L; ++l) {
            const int N = p.out[l];
            const int cw = N / 4;                       // 32 or 64 columns: one or two passes
            float bias[2];
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                const int c = group * cw + 32 * q + lane;
                bias[q] = 32 * q < cw ? __ldg(p.bias[l] + c) : 0.f;
            }
            if (!mbar_wait_idle(smem_u32(acc_full), l & 1, abort_flag)) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
            __nv_bfloat16* Y = static_cast<__nv_bfloat16*>(p.Y[l]);
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                if (32 * q >= cw) break;
                const int c0 = group * cw + 32 * q;
                float v[32];
                tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)c0, v);
                uint32_t u[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const float x0 = fmaxf(v[2 * j] + __shfl_sync(0xffffffffu, bias[q], 2 * j), 0.f);
                    const float x1 = fmaxf(v[2 * j + 1] + __shfl_sync(0xffffffffu, bias[q], 2 * j + 1), 0.f);
                    u[j] = pack_bf16(x0, x1);
                }
                // this row's 32 columns to global memory, through the staging buffer
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    sts128(stage_unit(stage, lane, c), make_uint4(u[4 * c], u[4 * c + 1], u[4 * c + 2], u[4 * c + 3]));
                __syncwarp();
                store_bf16_block(stage, lane, Y, p.ldy[l], nullptr, nomask, r0, p.M, c0, 32);
                __syncwarp();
                // and into the activation tile as the next layer's A operand: k-block c0 / 64, 16-byte chunks
                // (c0 mod 64) / 8 + j of this row's 128 bytes, swizzled by row mod 8
                if (l + 1 < L) {
                    const uint32_t rowb = smem_u32(act + (c0 / BK) * CH_KB_BYTES) + (uint32_t)row * 128u;
                    const int ch0 = (c0 % BK) / 8;
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        sts128(rowb + (uint32_t)((((ch0 + j) ^ (row & 7)) & 7) << 4),
                               make_uint4(u[4 * j], u[4 * j + 1], u[4 * j + 2], u[4 * j + 3]));
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(act_ready));
        }
    }
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) atomicOr(p.err, ST_KERNEL_TIMEOUT);
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(256) : "memory");
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

int sm_count() {
    static int n = 0;
    static std::once_flag once;
    std::call_once(once, [] {
        int dev = 0, v = 0;
        if (cudaGetDevice(&dev) == cudaSuccess &&
            cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && v > 0)
            n = v;
        else
            n = 148;
        cudaGetLastError();
    });
    return n;
}

template <typename K>
cudaError_t set_smem(K kernel, size_t bytes, bool cluster) {
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, (int)cudaSharedmemCarveoutMaxShared);
    if (e == cudaSuccess && cluster) e = cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    return e;
}

// Relative cost of one 128 x BN tile's k-block: 128-wide tiles read A and B from shared memory
// for half the MMA work of 256-wide ones.
constexpr double kCost128 = 0.62, kCost256 = 1.0;
constexpr long long kMinTiles256 = 48;

// Shared-memory sizes (and cluster sizes past 8) the kernels need, set once.
cudaError_t kernel_attrs() {
    static cudaError_t attr = [] {
        cudaError_t e = set_smem(tc_gemm_kernel<128>, GemmCfg<128>::SMEM, false);
        if (e == cudaSuccess) e = set_smem(tc_gemm_kernel<256>, GemmCfg<256>::SMEM, false);
        if (e == cudaSuccess) e = set_smem(tc_dw_kernel, DwCfg::SMEM, true);
        if (e == cudaSuccess) e = set_smem(tc_chain_kernel, CH_SMEM, false);
        return e;
    }();
    return attr;
}

}  // namespace

bool tc_chain_supported(int L, int K0, const int* out) {
    if (L < 2 || L > CH_MAX_LAYERS || K0 < 1 || K0 > 4 * BK) return false;
    for (int l = 0; l < L; ++l)
        if (out[l] != 128 && out[l] != 256) return false;
    return tc_available();
}

cudaError_t launch_tc_chain(const TcChain& c, cudaStream_t s) {
    int outs[CH_MAX_LAYERS];
    for (int l = 0; l < c.L && l < CH_MAX_LAYERS; ++l) outs[l] = c.out[l];
    if (!tc_chain_supported(c.L, c.K0, outs) || c.M < 1) return cudaErrorInvalidValue;
    const cudaError_t attr = kernel_attrs();
    if (attr != cudaSuccess) return attr;
    ChainMaps maps;
    std::memset(&maps, 0, sizeof maps);
    ChainParams p;
    std::memset(&p, 0, sizeof p);
    bool ok = make_map(&maps.x, c.X, c.ldx, c.M, c.ldx, BK, BM);
    for (int l = 0; l < c.L; ++l) {
        const int in = l == 0 ? c.K0 : c.out[l - 1];
        ok &= c.ldw[l] >= in && make_map(&maps.w[l], c.W[l], c.ldw[l], c.out[l], c.ldw[l], BK, c.out[l]);
        p.out[l] = c.out[l];
        p.bias[l] = c.bias[l];
        p.Y[l] = c.Y[l];
        p.ldy[l] = c.ldy[l];
    }
    if (!ok) return cudaErrorInvalidValue;
    p.L = c.L;
    p.M = c.M;
    p.K0 = c.K0;
    p.err = c.err;
    p.hdr = c.hdr;
    tc_chain_kernel<<<(c.M + BM - 1) / BM, GEMM_THREADS, CH_SMEM, s>>>(maps, p);
    return cudaGetLastError();
}

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
    return !(concat && kb % DW_BN != 0);
}

bool tc_supported_dw(int out, int in, bool concat, int kb) { return tc_shape_dw(out, in, concat, kb) && tc_available(); }

void tc_choose_split(int out, int in, int rows, int* nsplit, int* kchunk) {
    // the cluster reduces its ranks' partials: one reduced gradient per layer
    (void)out;
    (void)in;
    *nsplit = 1;
    *kchunk = rows;
}

namespace {

// How many clusters of `cs` weight-gradient CTAs this device can run at once (its SMs per GPC and the
// kernel's shared memory decide); 0 when such a cluster cannot be scheduled.
int active_clusters(int cs) {
    static int cache[5];
    static std::once_flag once;
    std::call_once(once, [] {
        for (int j = 0; j < 5; ++j) cache[j] = 0;
        if (kernel_attrs() != cudaSuccess) return;
        for (int j = 0; j < 5; ++j) {
            const int c = 1 << j;
            cudaLaunchConfig_t lc;
            std::memset(&lc, 0, sizeof lc);
            lc.gridDim = dim3(c, 1, 1);
            lc.blockDim = dim3(THREADS, 1, 1);
            lc.dynamicSmemBytes = DwCfg::SMEM;
            cudaLaunchAttribute at[1];
            at[0].id = cudaLaunchAttributeClusterDimension;
            at[0].val.clusterDim.x = c;
            at[0].val.clusterDim.y = 1;
            at[0].val.clusterDim.z = 1;
            lc.attrs = at;
            lc.numAttrs = 1;
            int n = 0;
            const cudaError_t e = cudaOccupancyMaxActiveClusters(&n, tc_dw_kernel, &lc);
            cudaGetLastError();
            cache[j] = e == cudaSuccess ? n : 0;
        }
    });
    int j = 0;
    while ((1 << j) < cs && j < 4) ++j;
    return cache[j];
}

// Workspace floats a cs-rank weight-gradient launch exchanges its partials through.
long long dw_ws_need(int out, int in, int cs) {
    const long long tm = (out + BM - 1) / BM, tn = (in + DW_BN - 1) / DW_BN;
    return (long long)cs * tm * tn * BM * DW_BN + (long long)cs * tm * BM;
}

}  // namespace

long long tc_dw_ws_floats(int out, int in, int rows) {
    const int stages = (rows + DW_KS - 1) / DW_KS;
    const int cs_max = std::min(MAX_CLUSTER, std::max(1, stages / 2));
    return dw_ws_need(out, in, cs_max);
}

// Cluster size of the weight gradient: the one with the least estimated time, counting the waves of
// clusters the device can co-schedule, the 128-row stages each rank streams (about 0.33 us each, bound by
// their four TMA boxes) and a fixed cost per CTA (set-up, exchange, epilogue) of about 2.5 us; ranks keep
// at least kDwMinStages stages, the kernel spreads over at most kDwMaxCtas CTAs (the worker streams' kernels
// share the SMs: a weight gradient that holds fewer SMs a little longer leaves more to the others, which
// measured faster on every bf16 workload) and the exchange fits the workspace.  The tile width is 128.
constexpr long long kDwMaxCtas = 64;   // CTAs a weight gradient may spread over
constexpr int kDwMinStages = 4;       // 128-row stages each rank streams at least
void tc_dw_plan(int out, int in, int rows, bool concat, int kb, long long ws_floats, int* bn_out, int* cs_out) {
    (void)concat;
    (void)kb;
    const int stages = std::max(1, (rows + DW_KS - 1) / DW_KS);
    const long long tiles = (long long)((out + BM - 1) / BM) * ((in + DW_BN - 1) / DW_BN);
    double best = 1e30;
    int bcs = 1;
    for (int cs = 1; cs <= MAX_CLUSTER; cs *= 2) {
        if (cs > 1 && stages < kDwMinStages * cs) break;
        if (cs > 1 && tiles * cs > kDwMaxCtas) break;
        if (dw_ws_need(out, in, cs) > ws_floats) break;
        const long long slots = cs == 1 ? (long long)sm_count() : active_clusters(cs);
        if (slots < 1) continue;
        const double waves = (double)((tiles + slots - 1) / slots);
        const double t = waves * ((double)((stages + cs - 1) / cs) * 0.33 + 2.5);
        if (t < best - 1e-9) {
            best = t;
            bcs = cs;
        }
    }
    *bn_out = DW_BN;
    *cs_out = bcs;
}

cudaError_t launch_tc_gemm(const TcGemm& g, cudaStream_t s) {
    const cudaError_t attr = kernel_attrs();
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
    if (g.mode == GEMM_DW) {
        // A(m = out, k = row) = D[row, out], B(n = in, k = row) = X[row, in]: both MN-major, boxes of
        // 64 columns by 128 rows
        int bn = DW_BN, cs = 1;
        tc_dw_plan(g.M, g.N, g.K, g.B2 != nullptr, g.kb, g.ws_floats, &bn, &cs);
        if (!g.ws || dw_ws_need(g.M, g.N, cs) > g.ws_floats) return cudaErrorInvalidValue;
        if (g.B2 && g.kb % DW_BN != 0) return cudaErrorInvalidValue;
        p.a_mn = 1;
        p.b_mn = 1;
        p.ka = 1 << 30;
        p.kb = g.B2 ? g.kb : (1 << 30);
        ok &= make_map(&ta, g.A, g.lda, g.K, g.lda, 64, DW_KS);
        const long long n1 = g.B2 ? g.kb : g.ldb;
        ok &= make_map(&tb, g.B, n1, g.K, g.ldb, 64, DW_KS);
        tb2 = tb;
        if (g.B2) ok &= make_map(&tb2, g.B2, g.ldb2, g.K, g.ldb2, 64, DW_KS);
        if (!ok) return cudaErrorInvalidValue;
        p.kchunk = ((g.K + cs - 1) / cs + DW_KS - 1) / DW_KS * DW_KS;
        p.P = g.P;
        p.ldp = g.ldc;
        p.Pb = g.Pb;
        p.ws = g.ws;
        p.Wm = g.Wm;
        p.bm = g.bm;
        p.cW = g.cW;
        p.cw_ld = g.cw_ld;
        p.cb = g.cb;
        p.lr = g.lr;
        p.tiles_m = (g.M + BM - 1) / BM;
        p.tiles_n = (g.N + DW_BN - 1) / DW_BN;
        p.wsb = g.ws + (long long)cs * p.tiles_m * p.tiles_n * BM * DW_BN;
        cudaLaunchConfig_t lc;
        std::memset(&lc, 0, sizeof lc);
        lc.gridDim = dim3(cs, p.tiles_n, p.tiles_m);
        lc.blockDim = dim3(THREADS, 1, 1);
        lc.dynamicSmemBytes = DwCfg::SMEM;
        lc.stream = s;
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = cs;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        lc.attrs = at;
        lc.numAttrs = 1;
        return cudaLaunchKernelEx(&lc, tc_dw_kernel, ta, tb, tb2, p);
    }
    // forward / input gradient: 256-wide tiles when they still give at least kMinTiles256 CTAs (they do twice
    // the work per TMA stage, so they take half the SM time of 128-wide ones: the step runs its worker
    // streams' kernels side by side), else unless 128-wide ones finish the grid in fewer cost-weighted
    // rounds of the SMs
    const int tm = (g.M + BM - 1) / BM;
    const long long t128 = (long long)tm * ((g.N + 127) / 128), t256 = (long long)tm * ((g.N + 255) / 256);
    const int sms = sm_count();
    const double c128 = (double)((t128 + sms - 1) / sms) * kCost128;
    const double c256 = (double)((t256 + sms - 1) / sms) * kCost256;
    const int bn = (g.N > 128 && (t256 >= kMinTiles256 || c256 <= c128)) ? 256 : 128;
    p.tiles_m = tm;
    p.tiles_n = (g.N + bn - 1) / bn;
    if (g.mode == GEMM_FWD) {
        // A = X [rows, K] (two maps when concatenated along K), B = W [out, K]
        p.a_mn = 0;
        p.b_mn = 0;
        p.ka = g.A2 ? g.ka : (1 << 30);
        const long long k1 = g.A2 ? g.ka : g.lda;
        ok &= make_map(&ta, g.A, k1, g.M, g.lda, 64, BM);
        ta2 = ta;
        if (g.A2) ok &= make_map(&ta2, g.A2, g.lda2, g.M, g.lda2, 64, BM);
        ok &= make_map(&tb, g.B, g.ldb, g.N, g.ldb, 64, bn);
        p.bias = g.bias;
        p.relu = g.relu;
        p.C = g.C;
        p.ldc = g.ldc;
    } else {
        // A = D [rows, K = out], B(n, k) = W[k, n]: W [out rows, in_ld] is MN-major
        p.a_mn = 0;
        p.b_mn = 1;
        p.ka = 1 << 30;
        ok &= make_map(&ta, g.A, g.lda, g.M, g.lda, 64, BM);
        ta2 = ta;
        ok &= make_map(&tb, g.B, g.ldb, g.K, g.ldb, 64, 64);
        p.C = g.C;
        p.ldc = g.ldc;
        p.mask1 = g.mask1;
        p.n_split = g.n_split;
        p.C2 = g.C2;
        p.ldc2 = g.ldc2;
        p.c2_f32 = g.c2_f32;
        p.mask2 = g.mask2;
    }
    if (!ok) return cudaErrorInvalidValue;
    const long long tiles = (long long)p.tiles_m * p.tiles_n;
    const int grid = (int)std::min<long long>(tiles, sms);
    if (bn == 256)
        tc_gemm_kernel<256><<<grid, GEMM_THREADS, GemmCfg<256>::SMEM, s>>>(ta, ta2, tb, p);
    else
        tc_gemm_kernel<128><<<grid, GEMM_THREADS, GemmCfg<128>::SMEM, s>>>(ta, ta2, tb, p);
    return cudaGetLastError();
}

}  // namespace vfl
