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

// The same selection with the keys in registers (lane l holds the keys of labels l + 32 m,
// 0 for labels >= Tb): an MSB-first radix walk over ballots narrows the keys whose high bits
// equal a prefix to the group that holds the keep-th largest key; keys above the group are
// kept, and within it the largest ones, the first equal ones in label order. The walk stops as
// soon as the group holds exactly the keys still to keep (all of it is then kept; for random
// scores after about a dozen of the 32 bits). Same total order, so the same lists as
// rank_select; kPer ballots a round instead of Tb shared-memory reads.
template <int kPer>
__device__ __forceinline__ void ballot_select(const uint32_t (&key)[kPer], int Tb, int keep, int lane, int32_t* dst)
{
    bool valid[kPer];
#pragma unroll
    for (int m = 0; m < kPer; ++m) valid[m] = lane + 32 * m < Tb;
    uint32_t prefix = 0u, pmask = 0u;
    int remaining = keep, group = Tb;  // keys still to keep; keys whose bits under pmask equal prefix
    for (int bit = 31; bit >= 0 && group != remaining; --bit) {
        const uint32_t trial = prefix | (1u << bit), tmask = pmask | (1u << bit);
        int c = 0;
#pragma unroll
        for (int m = 0; m < kPer; ++m) c += __popc(__ballot_sync(0xffffffffu, valid[m] && (key[m] & tmask) == trial));
        if (c >= remaining) {
            prefix = trial;
            group = c;
        } else {
            remaining -= c;
            group -= c;
        }
        pmask = tmask;
    }
    int out = 0, eq_seen = 0;
#pragma unroll
    for (int m = 0; m < kPer; ++m) {
        const uint32_t hi = key[m] & pmask;
        const bool gt = valid[m] && hi > prefix, eq = valid[m] && hi == prefix;
        const uint32_t eqm = __ballot_sync(0xffffffffu, eq);
        const int eq_rank = eq_seen + __popc(eqm & ((1u << lane) - 1u));
        const bool kept = gt || (eq && eq_rank < remaining);
        const uint32_t km = __ballot_sync(0xffffffffu, kept);
        if (kept) dst[out + __popc(km & ((1u << lane) - 1u))] = lane + 32 * m;
        out += __popc(km);
        eq_seen += __popc(eqm);
    }
}

}  // namespace sel
}  // namespace ssba
