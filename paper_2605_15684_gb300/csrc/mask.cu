// mask.cu -- block compression, affinity and Top-k gating (Sec. 2.2; Algorithm 1,
// partition .. Top-k Smallest) as two HBM-friendly kernels:
//
//   ssba_pool_kernel    one CTA per (batch*head, block): gathers the block's 64
//                       shifted tokens of Q and K with 16-byte loads, and writes the
//                       fp32 block means q_b, k_b (Eq. for q_b/k_b) to the workspace.
//                       Dominant cost: reading Q and K once (algorithmic bytes
//                       2 * B * heads * N * head_dim * elem).
//   ssba_select_kernel  one warp per query block: S row = q_b[i] . k_b[j] for all j in
//                       fp32, then an exact radix select of the `keep` largest entries
//                       under the total order (S descending, label ascending), i.e. the
//                       k_drop smallest are dropped and ties keep the lower label; the
//                       kept labels are written in ascending order.
#include <cstdio>

#include "common.cuh"

namespace ssba {

namespace {

constexpr int kPoolThreads = 128;

template <typename T>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
    static constexpr int kElems = 8;  // 16 bytes
    __device__ static void to_f32(const uint4& v, float* out)
    {
        const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float2 f = __bfloat1622float2(p[i]);
            out[2 * i] = f.x;
            out[2 * i + 1] = f.y;
        }
    }
};
template <>
struct Vec<float> {
    static constexpr int kElems = 4;
    __device__ static void to_f32(const uint4& v, float* out)
    {
        out[0] = __uint_as_float(v.x);
        out[1] = __uint_as_float(v.y);
        out[2] = __uint_as_float(v.z);
        out[3] = __uint_as_float(v.w);
    }
};

// smem: tokens of the block staged in fp32, [2 tensors][blk*blk][d]; column sums are
// then taken in in-block position order (a deterministic order).
template <typename T>
__global__ void __launch_bounds__(kPoolThreads) ssba_pool_kernel(const T* __restrict__ Q,
                                                                 const T* __restrict__ K, Grid g, int d,
                                                                 float* __restrict__ qb,
                                                                 float* __restrict__ kb)
{
    extern __shared__ float stage[];  // [2][P][d]
    const int label = blockIdx.x;
    const int bh = blockIdx.y;
    const int P = g.blk * g.blk;
    const int N = g.H * g.W;
    constexpr int VE = Vec<T>::kElems;
    const int cpr = d / VE;  // 16-byte chunks per token row
    const int chunks = P * cpr;
    const T* Qh = Q + (size_t)bh * N * d;
    const T* Kh = K + (size_t)bh * N * d;

    for (int ci = threadIdx.x; ci < 2 * chunks; ci += kPoolThreads) {
        int which = ci >= chunks;
        int cc = which ? ci - chunks : ci;
        int pos = cc / cpr, col = cc - pos * cpr;
        int tok = g.token(label, pos);
        const T* src = (which ? Kh : Qh) + (size_t)tok * d + col * VE;
        uint4 v = __ldg(reinterpret_cast<const uint4*>(src));
        float f[VE];
        Vec<T>::to_f32(v, f);
        float* dst = stage + ((size_t)which * P + pos) * d + col * VE;
#pragma unroll
        for (int e = 0; e < VE; ++e) dst[e] = f[e];
    }
    __syncthreads();
    const float inv = 1.0f / (float)P;
    for (int t = threadIdx.x; t < 2 * d; t += kPoolThreads) {
        int which = t >= d;
        int c = which ? t - d : t;
        const float* src = stage + (size_t)which * P * d + c;
        float acc = 0.f;
        for (int pos = 0; pos < P; ++pos) acc += src[(size_t)pos * d];
        float* out = which ? kb : qb;
        out[((size_t)bh * g.Tb() + label) * d + c] = acc * inv;
    }
}

constexpr int kSelWarps = 8;
constexpr int kSelKeyChunk = 256;
constexpr int kMaxTb = 2048;

__device__ __forceinline__ uint32_t order_key(float s)
{
    float f = s + 0.0f;  // -0.0 -> +0.0 so that equal values compare equal
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// smem: kbT [d][kSelKeyChunk] | q rows [kSelWarps][d] | S rows [kSelWarps][Tb]
__global__ void __launch_bounds__(kSelWarps * 32) ssba_select_kernel(const float* __restrict__ qb,
                                                                     const float* __restrict__ kb, int Tb,
                                                                     int d, int keep,
                                                                     int32_t* __restrict__ idx,
                                                                     int32_t* __restrict__ cnt,
                                                                     float* __restrict__ scores)
{
    extern __shared__ float sm[];
    float* kbT = sm;
    float* qs = kbT + (size_t)d * kSelKeyChunk;
    float* Srow = qs + (size_t)kSelWarps * d;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int bh = blockIdx.y;
    const int row = blockIdx.x * kSelWarps + warp;
    const bool active = row < Tb;
    const float* kbh = kb + (size_t)bh * Tb * d;
    float* S = Srow + (size_t)warp * Tb;

    if (active)
        for (int c = lane; c < d; c += 32) qs[warp * d + c] = qb[((size_t)bh * Tb + row) * d + c];

    // S row in key chunks: kbT holds a transposed chunk so lanes read consecutive keys.
    for (int j0 = 0; j0 < Tb; j0 += kSelKeyChunk) {
        const int nk = min(kSelKeyChunk, Tb - j0);
        __syncthreads();
        for (int e = threadIdx.x; e < nk * d; e += kSelWarps * 32) {
            int j = e / d, c = e - j * d;
            kbT[c * kSelKeyChunk + j] = kbh[(size_t)(j0 + j) * d + c];
        }
        __syncthreads();
        if (active) {
            for (int j = lane; j < nk; j += 32) {
                float acc = 0.f;
                for (int c = 0; c < d; ++c) acc = fmaf(qs[warp * d + c], kbT[c * kSelKeyChunk + j], acc);
                S[j0 + j] = acc;
            }
        }
    }
    __syncwarp();
    if (!active) return;

    const size_t rowoff = (size_t)bh * Tb + row;
    if (scores)
        for (int j = lane; j < Tb; j += 32) scores[rowoff * Tb + j] = S[j];

    // keep-th largest key by MSB-first radix select
    uint32_t prefix = 0, pmask = 0;
    int remaining = keep;
    for (int bit = 31; bit >= 0; --bit) {
        const uint32_t trial = prefix | (1u << bit), tmask = pmask | (1u << bit);
        int c = 0;
        for (int j = lane; j < Tb; j += 32) c += (order_key(S[j]) & tmask) == trial;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
        if (c >= remaining) prefix = trial;
        else remaining -= c;
        pmask = tmask;
    }
    // kept: key > T, or key == T among the first `remaining` equal ones (lowest labels)
    const uint32_t T = prefix;
    int out = 0, eq_seen = 0;
    int32_t* dst = idx + rowoff * keep;
    for (int j0 = 0; j0 < Tb; j0 += 32) {
        const int j = j0 + lane;
        uint32_t key = j < Tb ? order_key(S[j]) : 0u;
        bool gt = j < Tb && key > T;
        bool eq = j < Tb && key == T;
        uint32_t eqm = __ballot_sync(0xffffffffu, eq);
        int eq_rank = eq_seen + __popc(eqm & ((1u << lane) - 1u));
        bool kept = gt || (eq && eq_rank < remaining);
        uint32_t km = __ballot_sync(0xffffffffu, kept);
        if (kept) dst[out + __popc(km & ((1u << lane) - 1u))] = j;
        out += __popc(km);
        eq_seen += __popc(eqm);
    }
    if (lane == 0) cnt[rowoff] = keep;
}

}  // namespace

int launch_pool(const ssba_desc& d, const Grid& g, const void* Q, const void* K, float* qb, float* kb,
                cudaStream_t st)
{
    const int P = g.blk * g.blk;
    size_t smem = (size_t)2 * P * d.head_dim * sizeof(float);
    dim3 grid(g.Tb(), d.B * d.heads);
    if (smem > 200 * 1024) {
        set_error("ssba_build_mask: block*block*head_dim too large for the pooling kernel");
        return SSBA_ERR_UNSUPPORTED;
    }
    if (d.dtype == SSBA_BF16) {
        auto k = ssba_pool_kernel<__nv_bfloat16>;
        if (smem > 48 * 1024) cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        k<<<grid, kPoolThreads, smem, st>>>(static_cast<const __nv_bfloat16*>(Q),
                                            static_cast<const __nv_bfloat16*>(K), g, d.head_dim, qb, kb);
    } else {
        auto k = ssba_pool_kernel<float>;
        if (smem > 48 * 1024) cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        k<<<grid, kPoolThreads, smem, st>>>(static_cast<const float*>(Q), static_cast<const float*>(K), g,
                                            d.head_dim, qb, kb);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("ssba_pool_kernel launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

int launch_select(const ssba_desc& d, const Grid& g, int keep, const float* qb, const float* kb,
                  int32_t* idx, int32_t* cnt, float* scores, cudaStream_t st)
{
    const int Tb = g.Tb();
    if (Tb > kMaxTb) {
        set_error("ssba_build_mask: Tb=%d exceeds the selection kernel's limit of %d blocks", Tb, kMaxTb);
        return SSBA_ERR_UNSUPPORTED;
    }
    size_t smem = ((size_t)d.head_dim * kSelKeyChunk + (size_t)kSelWarps * d.head_dim +
                   (size_t)kSelWarps * Tb) * sizeof(float);
    if (smem > 220 * 1024) {
        set_error("ssba_build_mask: selection working set too large (%zu bytes)", smem);
        return SSBA_ERR_UNSUPPORTED;
    }
    if (smem > 48 * 1024)
        cudaFuncSetAttribute(ssba_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    dim3 grid((Tb + kSelWarps - 1) / kSelWarps, d.B * d.heads);
    ssba_select_kernel<<<grid, kSelWarps * 32, smem, st>>>(qb, kb, Tb, d.head_dim, keep, idx, cnt, scores);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("ssba_select_kernel launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

}  // namespace ssba
