// attn_simt.cu -- fp32 block-sparse attention forward on CUDA cores (Sec. 2.2
// Efficient Sparse Execution; Algorithm 1 SparseAttention over the expanded mask).
//
// One CTA per (batch*head, query block), two threads per query row: each thread
// owns the interleaved half {h, h+2, ...} of head_dim (so the two halves hit
// adjacent shared-memory banks). The kept key blocks are visited in list order;
// each block's K and V rows (gathered through the shifted grid, any shift) are
// staged in shared memory and folded into an online softmax in fp32 with expf.
// This path serves fp32 inputs, where the tensor-core path's bf16 operands would
// not meet fp32 accuracy.
#include "common.cuh"

namespace ssba {

namespace {

constexpr int kD = 64;             // head_dim of this kernel
constexpr int kP = 64;             // tokens per block (8 x 8)
constexpr int kThreads = 2 * kP;   // two threads per query row

__global__ void __launch_bounds__(kThreads) ssba_attn_simt_f32_kernel(
    const float* __restrict__ Q, const float* __restrict__ K, const float* __restrict__ V, Grid g, int keep,
    float scale, const int32_t* __restrict__ idx, const int32_t* __restrict__ cnt, float* __restrict__ O,
    float* __restrict__ lse)
{
    __shared__ float Ks[kP][kD];
    __shared__ float Vs[kP][kD];
    const int label = blockIdx.x, bh = blockIdx.y;
    const int Tb = g.Tb();
    const int N = g.H * g.W;
    const int r = threadIdx.x >> 1, h = threadIdx.x & 1;
    const int tok = g.token(label, r);
    const float* Qh = Q + (size_t)bh * N * kD;
    const float* Kh = K + (size_t)bh * N * kD;
    const float* Vh = V + (size_t)bh * N * kD;

    float q[kD / 2], o[kD / 2];
#pragma unroll
    for (int c = 0; c < kD / 2; ++c) {
        q[c] = Qh[(size_t)tok * kD + 2 * c + h];
        o[c] = 0.f;
    }
    float m = -INFINITY, l = 0.f;
    const int32_t* list = idx + ((size_t)bh * Tb + label) * keep;
    const int nblk = min(max(cnt[(size_t)bh * Tb + label], 0), keep);

    for (int t = 0; t < nblk; ++t) {
        const int j = list[t];
        if ((unsigned)j >= (unsigned)Tb) continue;  // malformed label: skipped, never read out of bounds
        __syncthreads();
        for (int e = threadIdx.x; e < kP * (kD / 4); e += kThreads) {
            int p = e / (kD / 4), c4 = e - p * (kD / 4);
            int kt = g.token(j, p);
            reinterpret_cast<float4*>(&Ks[p][0])[c4] =
                __ldg(reinterpret_cast<const float4*>(Kh + (size_t)kt * kD) + c4);
            reinterpret_cast<float4*>(&Vs[p][0])[c4] =
                __ldg(reinterpret_cast<const float4*>(Vh + (size_t)kt * kD) + c4);
        }
        __syncthreads();
        float s[kP];
        float bmax = -INFINITY;
#pragma unroll 8
        for (int p = 0; p < kP; ++p) {
            float acc = 0.f;
#pragma unroll
            for (int c = 0; c < kD / 2; ++c) acc = fmaf(q[c], Ks[p][2 * c + h], acc);
            acc += __shfl_xor_sync(0xffffffffu, acc, 1);
            s[p] = acc * scale;
            bmax = fmaxf(bmax, s[p]);
        }
        const float mnew = fmaxf(m, bmax);
        const float alpha = expf(m - mnew);  // 0 on the first block (m = -inf)
        l *= alpha;
#pragma unroll
        for (int c = 0; c < kD / 2; ++c) o[c] *= alpha;
#pragma unroll 8
        for (int p = 0; p < kP; ++p) {
            const float pr = expf(s[p] - mnew);
            l += pr;
#pragma unroll
            for (int c = 0; c < kD / 2; ++c) o[c] = fmaf(pr, Vs[p][2 * c + h], o[c]);
        }
        m = mnew;
    }
    const float inv = l > 0.f ? 1.f / l : 0.f;  // an empty list gives O = 0, lse = -inf
    float* Oh = O + (size_t)bh * N * kD + (size_t)tok * kD;
#pragma unroll
    for (int c = 0; c < kD / 2; ++c) Oh[2 * c + h] = o[c] * inv;
    if (h == 0) lse[(size_t)bh * N + tok] = l > 0.f ? m + logf(l) : -INFINITY;
}

}  // namespace

int launch_attn_simt_f32(const ssba_desc& d, const Grid& g, int keep, float scale, const float* Q,
                         const float* K, const float* V, const int32_t* idx, const int32_t* cnt, float* O,
                         float* lse, cudaStream_t st)
{
    if (d.head_dim != kD || g.blk * g.blk != kP) {
        set_error("ssba_forward (fp32): needs head_dim=%d and block=8", kD);
        return SSBA_ERR_UNSUPPORTED;
    }
    dim3 grid(g.Tb(), d.B * d.heads);
    ssba_attn_simt_f32_kernel<<<grid, kThreads, 0, st>>>(Q, K, V, g, keep, scale, idx, cnt, O, lse);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("ssba_attn_simt_f32_kernel launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

}  // namespace ssba
