// select.cuh -- the Top-k gating of Sec. 2.2 / Algorithm 1 ("Top-k Smallest" dropped) on one
// row of affinities, shared by the mask kernels and the attention kernel's in-kernel
// selection, so that both keep bit-identical lists for the same scores.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

namespace ssba {
namespace sel {

// Order-preserving unsigned key of a float: larger key = larger value; -0.0 == +0.0.
__device__ __forceinline__ uint32_t order_key(float s)
{
    float f = s + 0.0f;  // -0.0 -> +0.0 so that equal values compare equal
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Kept labels of one row by rank counting; lane l owns labels l + 32m, m < kPer.
template <int kPer>
__device__ __forceinline__ void rank_select(const uint32_t* S, int Tb, int keep, int lane, int32_t* dst)
{
    uint32_t mine[kPer];
    int rank[kPer];
#pragma unroll
    for (int m = 0; m < kPer; ++m) {
        const int j = lane + 32 * m;
        mine[m] = j < Tb ? S[j] : 0u;
        rank[m] = 0;
    }
#pragma unroll 8
    for (int k = 0; k < Tb; ++k) {
        const uint32_t v = S[k];  // broadcast read
#pragma unroll
        for (int m = 0; m < kPer; ++m) rank[m] += (v > mine[m]) || (v == mine[m] && k < lane + 32 * m);
    }
    int out = 0;
#pragma unroll
    for (int m = 0; m < kPer; ++m) {
        const int j = lane + 32 * m;
        const bool kept = j < Tb && rank[m] < keep;
        const uint32_t km = __ballot_sync(0xffffffffu, kept);
        if (kept) dst[out + __popc(km & ((1u << lane) - 1u))] = j;
        out += __popc(km);
    }
}

}  // namespace sel
}  // namespace ssba
