// Philox4x32-10 counter-based normals for the DP mechanisms (device side).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace vfl {

// Philox4x32-10 (Salmon et al., SC'11): ten rounds of two 32x32->64 products,
// key bumped by the Weyl increments between rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 key) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const unsigned lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
        const unsigned lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
        c = make_uint4(hi1 ^ c.y ^ key.x, lo1, hi0 ^ c.w ^ key.y, lo0);
        key.x += 0x9E3779B9u;
        key.y += 0xBB67AE85u;
    }
    return c;
}

// Four N(0,1) draws for columns 4q..4q+3 of row r at step k: Philox4x32-10 block (q, r, k, tag) under
// key, words (x0, x1) and (x2, x3) through Box-Muller with u1 = ((x >> 8) + 1) 2^-24, u2 = (y >> 8) 2^-24.
__device__ __forceinline__ void dp_normals4(int q, int r, long long k, unsigned tag, uint2 key, float z[4]) {
    const uint4 w = philox4x32_10(make_uint4((unsigned)q, (unsigned)r, (unsigned)(k & 0xFFFFFFFFll), tag), key);
    const unsigned xs[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int p = 0; p < 2; ++p) {
        const float u1 = (float)((xs[2 * p] >> 8) + 1u) * 0x1p-24f;
        const float u2 = (float)(xs[2 * p + 1] >> 8) * 0x1p-24f;
        const float rad = sqrtf(-2.0f * logf(u1));
        float sn, cs;
        sincospif(2.0f * u2, &sn, &cs);
        z[2 * p] = rad * cs;
        z[2 * p + 1] = rad * sn;
    }
}

}  // namespace vfl
