// attn_bwd.cu -- gradients of the block-sparse attention (the backward pass of Algorithm 1's
// SparseAttention over the same kept blocks), on CUDA cores in fp32.
//
// For the output gradient dO, with p_nm = exp(scale q_n.k_m - lse_n) over the allowed pairs:
//   D_n  = dO_n . O_n
//   dV_m = sum_n p_nm dO_n
//   ds_nm = p_nm (dO_n . v_m - D_n)
//   dQ_n = scale sum_m ds_nm k_m,   dK_m = scale sum_n ds_nm q_n.
// Two kernels, no atomics, deterministic:
//   ssba_bwd_dq_kernel    one CTA per (batch*head, query block): two threads per query row
//                         (interleaved halves of head_dim, as the fp32 forward), the kept key
//                         blocks staged in shared memory in list order; writes dQ and D.
//   ssba_bwd_dkdv_kernel  one CTA per (batch*head, key block): finds, in ascending order, the
//                         query blocks whose lists hold it, stages each one's Q and dO, and
//                         accumulates dK and dV for its 64 key rows (two threads per row).
#include "common.cuh"

namespace ssba {

namespace {

constexpr int kD = 64;            // head_dim of these kernels
constexpr int kP = 64;            // tokens per block (8 x 8)
constexpr int kThreads = 2 * kP;  // two threads per row

__device__ __forceinline__ float ld_f32(const float* p) { return __ldg(p); }
__device__ __forceinline__ float ld_f32(const __nv_bfloat16* p) { return __bfloat162float(*p); }

// Stages rows g.token(label, p) of X (64 x 64, any dtype) as fp32 into dst.
template <typename T>
__device__ __forceinline__ void stage_block(float (*dst)[kD], const T* X, const Grid& g, int label)
{
    for (int e = threadIdx.x; e < kP * kD; e += kThreads) {
        const int p = e / kD, c = e - p * kD;
        dst[p][c] = ld_f32(X + (size_t)g.token(label, p) * kD + c);
    }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) ssba_bwd_dq_kernel(
    const T* __restrict__ Q, const T* __restrict__ K, const T* __restrict__ V, const T* __restrict__ O,
    const float* __restrict__ lse, const T* __restrict__ dO, Grid g, int keep, float scale,
    const int32_t* __restrict__ idx, const int32_t* __restrict__ cnt, float* __restrict__ dQ,
    float* __restrict__ Dbuf)
{
    __shared__ float Ks[kP][kD];
    __shared__ float Vs[kP][kD];
    const int label = blockIdx.x, bh = blockIdx.y;
    const int Tb = g.Tb();
    const int N = g.H * g.W;
    const int r = threadIdx.x >> 1, h = threadIdx.x & 1;
    const int tok = g.token(label, r);
    const size_t row = (size_t)bh * N + tok;

    float q[kD / 2], go[kD / 2], dq[kD / 2];
    float D = 0.f;
#pragma unroll
    for (int c = 0; c < kD / 2; ++c) {
        q[c] = ld_f32(Q + row * kD + 2 * c + h);
        go[c] = ld_f32(dO + row * kD + 2 * c + h);
        D = fmaf(go[c], ld_f32(O + row * kD + 2 * c + h), D);
        dq[c] = 0.f;
    }
    D += __shfl_xor_sync(0xffffffffu, D, 1);
    const float L = lse[row];
    const int32_t* list = idx + ((size_t)bh * Tb + label) * keep;
    const int nblk = min(max(cnt[(size_t)bh * Tb + label], 0), keep);
    for (int t = 0; t < nblk; ++t) {
        const int j = list[t];
        if ((unsigned)j >= (unsigned)Tb) continue;  // malformed label: skipped, never read out of bounds
        __syncthreads();
        stage_block(Ks, K + (size_t)bh * N * kD, g, j);
        stage_block(Vs, V + (size_t)bh * N * kD, g, j);
        __syncthreads();
#pragma unroll 4
        for (int p = 0; p < kP; ++p) {
            float s = 0.f, dp = 0.f;
#pragma unroll
            for (int c = 0; c < kD / 2; ++c) {
                s = fmaf(q[c], Ks[p][2 * c + h], s);
                dp = fmaf(go[c], Vs[p][2 * c + h], dp);
            }
            s += __shfl_xor_sync(0xffffffffu, s, 1);
            dp += __shfl_xor_sync(0xffffffffu, dp, 1);
            const float pr = expf(s * scale - L);
            const float ds = pr * (dp - D) * scale;
#pragma unroll
            for (int c = 0; c < kD / 2; ++c) dq[c] = fmaf(ds, Ks[p][2 * c + h], dq[c]);
        }
    }
#pragma unroll
    for (int c = 0; c < kD / 2; ++c) dQ[row * kD + 2 * c + h] = dq[c];
    if (h == 0) Dbuf[row] = D;
}

template <typename T>
__global__ void __launch_bounds__(kThreads) ssba_bwd_dkdv_kernel(
    const T* __restrict__ Q, const T* __restrict__ K, const T* __restrict__ V, const float* __restrict__ lse,
    const T* __restrict__ dO, const float* __restrict__ Dbuf, Grid g, int keep, float scale,
    const int32_t* __restrict__ idx, const int32_t* __restrict__ cnt, float* __restrict__ dK,
    float* __restrict__ dV)
{
    __shared__ float Qs[kP][kD];
    __shared__ float Gs[kP][kD];
    __shared__ float Ls[kP], Ds[kP];
    __shared__ int qlist[kThreads];
    __shared__ int wcount[kThreads / 32];
    const int label = blockIdx.x, bh = blockIdx.y;
    const int Tb = g.Tb();
    const int N = g.H * g.W;
    const int r = threadIdx.x >> 1, h = threadIdx.x & 1;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const size_t krow = (size_t)bh * N + g.token(label, r);

    float k[kD / 2], v[kD / 2], dk[kD / 2], dv[kD / 2];
#pragma unroll
    for (int c = 0; c < kD / 2; ++c) {
        k[c] = ld_f32(K + krow * kD + 2 * c + h);
        v[c] = ld_f32(V + krow * kD + 2 * c + h);
        dk[c] = 0.f;
        dv[c] = 0.f;
    }
    // query blocks whose lists hold this key block, in ascending order, kThreads at a time
    for (int i0 = 0; i0 < Tb; i0 += kThreads) {
        const int i = i0 + threadIdx.x;
        bool has = false;
        if (i < Tb) {
            const int32_t* list = idx + ((size_t)bh * Tb + i) * keep;
            const int n = min(max(cnt[(size_t)bh * Tb + i], 0), keep);
            for (int t = 0; t < n; ++t) has |= list[t] == label;
        }
        const unsigned b = __ballot_sync(0xffffffffu, has);
        __syncthreads();  // qlist / wcount of the previous round are consumed
        if (lane == 0) wcount[warp] = __popc(b);
        __syncthreads();
        int off = 0;
        for (int w = 0; w < warp; ++w) off += wcount[w];
        if (has) qlist[off + __popc(b & ((1u << lane) - 1u))] = i;
        int total = 0;
        for (int w = 0; w < kThreads / 32; ++w) total += wcount[w];
        __syncthreads();
        for (int u = 0; u < total; ++u) {
            const int qi = qlist[u];
            __syncthreads();
            stage_block(Qs, Q + (size_t)bh * N * kD, g, qi);
            stage_block(Gs, dO + (size_t)bh * N * kD, g, qi);
            if (threadIdx.x < kP) {
                const size_t qrow = (size_t)bh * N + g.token(qi, threadIdx.x);
                Ls[threadIdx.x] = lse[qrow];
                Ds[threadIdx.x] = Dbuf[qrow];
            }
            __syncthreads();
#pragma unroll 4
            for (int n = 0; n < kP; ++n) {
                float s = 0.f, dp = 0.f;
#pragma unroll
                for (int c = 0; c < kD / 2; ++c) {
                    s = fmaf(k[c], Qs[n][2 * c + h], s);
                    dp = fmaf(v[c], Gs[n][2 * c + h], dp);
                }
                s += __shfl_xor_sync(0xffffffffu, s, 1);
                dp += __shfl_xor_sync(0xffffffffu, dp, 1);
                const float pr = expf(s * scale - Ls[n]);
                const float ds = pr * (dp - Ds[n]) * scale;
#pragma unroll
                for (int c = 0; c < kD / 2; ++c) {
                    dv[c] = fmaf(pr, Gs[n][2 * c + h], dv[c]);
                    dk[c] = fmaf(ds, Qs[n][2 * c + h], dk[c]);
                }
            }
        }
    }
#pragma unroll
    for (int c = 0; c < kD / 2; ++c) {
        dK[krow * kD + 2 * c + h] = dk[c];
        dV[krow * kD + 2 * c + h] = dv[c];
    }
}

template <typename T>
int launch_bwd_t(const ssba_desc& d, const Grid& g, int keep, float scale, const void* Q, const void* K,
                 const void* V, const void* O, const float* lse, const void* dO, const int32_t* idx,
                 const int32_t* cnt, float* dQ, float* dK, float* dV, float* Dbuf, cudaStream_t st)
{
    dim3 grid(g.Tb(), d.B * d.heads);
    ssba_bwd_dq_kernel<T><<<grid, kThreads, 0, st>>>(
        static_cast<const T*>(Q), static_cast<const T*>(K), static_cast<const T*>(V), static_cast<const T*>(O), lse,
        static_cast<const T*>(dO), g, keep, scale, idx, cnt, dQ, Dbuf);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) {
        ssba_bwd_dkdv_kernel<T><<<grid, kThreads, 0, st>>>(
            static_cast<const T*>(Q), static_cast<const T*>(K), static_cast<const T*>(V), lse,
            static_cast<const T*>(dO), Dbuf, g, keep, scale, idx, cnt, dK, dV);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) {
        set_error("ssba_backward launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

}  // namespace

int launch_backward(const ssba_desc& d, const Grid& g, int keep, float scale, const void* Q, const void* K,
                    const void* V, const void* O, const float* lse, const void* dO, const int32_t* idx,
                    const int32_t* cnt, float* dQ, float* dK, float* dV, float* Dbuf, cudaStream_t st)
{
    if (d.head_dim != kD || g.blk * g.blk != kP) {
        set_error("ssba_backward: needs head_dim=%d and block=8", kD);
        return SSBA_ERR_UNSUPPORTED;
    }
    if (d.dtype == SSBA_BF16) {
        int rc = launch_backward_ws(d, g, keep, scale, Q, K, V, O, lse, dO, idx, cnt, dQ, dK, dV, Dbuf, st);
        if (rc != SSBA_ERR_UNSUPPORTED) return rc;
        rc = launch_backward_tc(d, g, keep, scale, Q, K, V, O, lse, dO, idx, cnt, dQ, dK, dV, Dbuf, st);
        if (rc != SSBA_ERR_UNSUPPORTED) return rc;
        return launch_bwd_t<__nv_bfloat16>(d, g, keep, scale, Q, K, V, O, lse, dO, idx, cnt, dQ, dK, dV, Dbuf, st);
    }
    return launch_bwd_t<float>(d, g, keep, scale, Q, K, V, O, lse, dO, idx, cnt, dQ, dK, dV, Dbuf, st);
}

}  // namespace ssba
