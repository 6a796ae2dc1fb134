// bwd_tile.cuh -- the 64 x 64 tile products and operand stores shared by the two tensor-core
// backward kernels (attn_bwd_tc.cu, attn_bwd_ws.cu). Tiles are 8 KB bf16, 128-byte swizzled
// (row r, 16-byte chunk c at chunk c ^ (r & 7)); every product is a tcgen05.mma kind::f16 of
// M=64 in four K=16 steps, issued by one thread.
#pragma once

#include "common.cuh"
#include "ptx.cuh"

namespace ssba {
namespace bwd {

constexpr int kD = 64;
constexpr int kT = 64;                   // tokens per block
constexpr uint32_t kTile = kT * kD * 2;  // 8 KB
constexpr uint32_t kIdescK = ptx::idesc_bf16_f32(64, 64, false, false);  // A, B K-major
constexpr uint32_t kIdescMN = ptx::idesc_bf16_f32(64, 64, false, true);  // B MN-major
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float fast_exp2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// C (64 x 64, fp32 TMEM at column `col`) = A B^T with A, B K-major 64 x 64 tiles in shared memory.
__device__ __forceinline__ void mma_kk(uint32_t col, uint32_t a, uint32_t b)
{
    const uint64_t ad = ptx::sdesc_sw128(a, 16, 1024), bd = ptx::sdesc_sw128(b, 16, 1024);
#pragma unroll
    for (int k = 0; k < 4; ++k) ptx::mma_ss(col, ad + (uint64_t)(k * 2), bd + (uint64_t)(k * 2), kIdescK, k > 0 ? 1u : 0u);
}

// C (+)= A B with A (64 x 64 bf16) a K-major shared tile and B a shared tile read MN-major
// (rows = the contraction index).
__device__ __forceinline__ void mma_sb(uint32_t col, uint32_t a, uint32_t b, bool accumulate)
{
    const uint64_t ad = ptx::sdesc_sw128(a, 16, 1024), bd = ptx::sdesc_sw128(b, 8192, 1024);
#pragma unroll
    for (int k = 0; k < 4; ++k)
        ptx::mma_ss(col, ad + (uint64_t)(k * 2), bd + (uint64_t)(k * 128), kIdescMN, (accumulate || k > 0) ? 1u : 0u);
}

// This thread's half row (row r of the M=64 data path, columns [32 h, 32 h + 32)) of a 64 x 64
// bf16 tile, 16 packed pairs, into the 128-byte-swizzled K-major layout at dst.
__device__ __forceinline__ void store_half_row(uint8_t* dst, int r, int h, const uint32_t (&v)[16])
{
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int c = 4 * h + i;
        *reinterpret_cast<uint4*>(dst + r * 128 + ((c ^ (r & 7)) << 4)) =
            make_uint4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
    }
}

// Arguments of the backward kernels (device pointers). ctr, toff, tcnt, tlist and ld are the
// persistent kernel's: its work counter, the transposed lists (CSR per head: for key block j of
// head bh, tcnt[bh Tb + j] query blocks, ascending, at tlist + toff[bh Tb + j]) and the row
// statistics by block; null for the per-block kernel.
struct BwdParams {
    const __nv_bfloat16 *Q, *K, *V, *O, *dO;
    const float* lse;
    const int32_t* idx;
    const int32_t* cnt;
    float *dQ, *dK, *dV, *Dbuf;
    int *ctr, *toff, *tcnt, *tlist;
    float2* ld;  // [B*heads][Tb][64]: (lse log2(e), D) of each block's rows in TMA tile order
    Grid g;
    int keep;
    float scale;
    int* status;
    uint64_t budget_ns;
    int withhold;  // failure-detection test hook: 1, CTA 0 announces its first pair's tiles
                   // and never copies them (ssba_test_backward_timeout)
};

// Byte offsets in the ssba_backward workspace: D of every row first (every path), then the
// persistent kernel's counter and transposed lists.
struct BwdLayout {
    size_t ctr, toff, tcnt, tlist, ld, bytes;
};
BwdLayout bwd_layout(const ssba_desc& d, const Grid& g, int keep);

// The row kernel: D for every row and, when p.tlist is set, the rows' (lse log2(e), D) by block
// in tile order, the counter reset and the transposed lists (one extra CTA per head). Launched plainly (it depends on all earlier work);
// the gradient kernel that follows is its programmatic dependent.
cudaError_t launch_bwd_rows(const BwdParams& p, int BH, cudaStream_t st);

}  // namespace bwd
}  // namespace ssba
