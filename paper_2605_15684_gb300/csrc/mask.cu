// mask.cu -- block compression, affinity and Top-k gating (Sec. 2.2; Algorithm 1,
// partition .. Top-k Smallest) as two HBM-friendly kernels:
//
//   ssba_pool_kernel    one CTA per (batch*head, block): gathers the block's 64 shifted
//                       tokens of Q and K with 16-byte loads, and writes the fp32 block
//                       means q_b, k_b (Eq. for q_b/k_b) to the workspace. Dominant cost:
//                       reading Q and K once (algorithmic bytes 2 * B * heads * N *
//                       head_dim * elem); HBM-bound.
//   ssba_select_kernel  one warp per query block: S row = q_b[i] . k_b[j] for all j in
//                       fp32, then an exact selection of the `keep` largest entries under
//                       the total order (S descending, label ascending), i.e. the k_drop
//                       smallest are dropped and ties keep the lower label; the kept labels
//                       are written in ascending order.
//   ssba_mask_fused_kernel  both steps in one launch for head_dim 64, 8x8 blocks and at
//                       most 256 blocks: a cluster of 8 CTAs per (batch, head) pools its
//                       blocks into shared memory, reads the head's k_b from the other CTAs
//                       of the cluster (distributed shared memory), and selects its rows
//                       (keys in registers, the radix walk of sel::ballot_select). No
//                       q_b/k_b round trip through global memory and no second launch.
#include <cooperative_groups.h>
#include <cstdio>

#include "common.cuh"
#include "ptx.cuh"
#include "select.cuh"

namespace ssba {

namespace {


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

// One CTA per (batch*head, block) for head_dim = 64, 256 threads: warp w reads tensor
// (w / 4 ? K : Q), rows [16 * (w % 4), +16) of the block. Lane l covers 16-byte chunk
// (l % 8) of rows l/8 + 4i, i < 4: four independent 16-byte loads per lane, so the whole
// block is requested in one round. Partial sums are combined in a fixed order (lanes by
// shuffles, warps through shared memory), then the block means are written.
template <typename T>
__global__ void __launch_bounds__(256) ssba_pool_kernel(const T* __restrict__ Q, const T* __restrict__ K, Grid g,
                                                        float* __restrict__ qb, float* __restrict__ kb)
{
    constexpr int kD = 64;
    constexpr int VE = Vec<T>::kElems;
    constexpr int CPR = kD / VE;            // 16-byte chunks per token row (8 bf16 / 16 fp32)
    constexpr int RPI = 32 / CPR;           // rows per warp instruction
    constexpr int ROWS = 16;                // rows per warp
    constexpr int LOADS = ROWS / RPI;       // loads per lane
    __shared__ float part[2][4][kD];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int which = warp >> 2, quarter = warp & 3;
    const int label = blockIdx.x, bh = blockIdx.y;
    const int N = g.H * g.W;
    const T* X = (which ? K : Q) + (size_t)bh * N * kD;
    const int col = lane % CPR, r0 = lane / CPR;
    uint4 v[LOADS];
#pragma unroll
    for (int i = 0; i < LOADS; ++i) {
        const int pos = quarter * ROWS + r0 + i * RPI;
        v[i] = __ldg(reinterpret_cast<const uint4*>(X + (size_t)g.token(label, pos) * kD + col * VE));
    }
    float acc[VE];
#pragma unroll
    for (int e = 0; e < VE; ++e) acc[e] = 0.f;
#pragma unroll
    for (int i = 0; i < LOADS; ++i) {
        float f[VE];
        Vec<T>::to_f32(v[i], f);
#pragma unroll
        for (int e = 0; e < VE; ++e) acc[e] += f[e];
    }
#pragma unroll
    for (int o = CPR; o < 32; o <<= 1)
#pragma unroll
        for (int e = 0; e < VE; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
    if (r0 == 0)
#pragma unroll
        for (int e = 0; e < VE; ++e) part[which][quarter][col * VE + e] = acc[e];
    __syncthreads();
    if (threadIdx.x < 2 * kD) {
        const int w = threadIdx.x >> 6, c = threadIdx.x & (kD - 1);
        const float sum = (part[w][0][c] + part[w][1][c]) + (part[w][2][c] + part[w][3][c]);
        (w ? kb : qb)[((size_t)bh * g.Tb() + label) * kD + c] = sum * (1.0f / 64.0f);
    }
}

// Generic-width fallback (any head_dim multiple of 16 bytes): the block's tokens are
// staged in fp32 in shared memory and column sums taken in in-block position order.
template <typename T>
__global__ void __launch_bounds__(128) ssba_pool_generic_kernel(const T* __restrict__ Q, const T* __restrict__ K,
                                                                Grid g, int d, float* __restrict__ qb,
                                                                float* __restrict__ kb)
{
    extern __shared__ float stage[];  // [2][P][d]
    const int label = blockIdx.x;
    const int bh = blockIdx.y;
    const int P = g.blk * g.blk;
    const int N = g.H * g.W;
    constexpr int VE = Vec<T>::kElems;
    const int cpr = d / VE;
    const int chunks = P * cpr;
    const T* Qh = Q + (size_t)bh * N * d;
    const T* Kh = K + (size_t)bh * N * d;
    for (int ci = threadIdx.x; ci < 2 * chunks; ci += 128) {
        int which = ci >= chunks;
        int cc = which ? ci - chunks : ci;
        int pos = cc / cpr, c = cc - pos * cpr;
        int tok = g.token(label, pos);
        uint4 v = __ldg(reinterpret_cast<const uint4*>((which ? Kh : Qh) + (size_t)tok * d + c * VE));
        float f[VE];
        Vec<T>::to_f32(v, f);
        float* dst = stage + ((size_t)which * P + pos) * d + c * VE;
#pragma unroll
        for (int e = 0; e < VE; ++e) dst[e] = f[e];
    }
    __syncthreads();
    const float inv = 1.0f / (float)P;
    for (int t = threadIdx.x; t < 2 * d; t += 128) {
        int which = t >= d;
        int c = which ? t - d : t;
        const float* src = stage + (size_t)which * P * d + c;
        float acc = 0.f;
        for (int pos = 0; pos < P; ++pos) acc += src[(size_t)pos * d];
        (which ? kb : qb)[((size_t)bh * g.Tb() + label) * d + c] = acc * inv;
    }
}

constexpr int kSelWarps = 8;
constexpr int kSelKeyChunk = 256;
constexpr int kMaxTb = 2048;
constexpr int kRankMaxTb = 256;  // rows up to this length use rank counting, longer ones radix select

// One warp per query block (row i of S), kSelWarps rows per CTA.
// smem: kbT [d][kSelKeyChunk + 1] (padded transpose of a key chunk) | q rows [kSelWarps][d]
//       | S rows as order keys [kSelWarps][Tb]
// S[i][j] = q_b[i] . k_b[j] in fp32 (FMA over d in order); the row is then reduced to its
// `keep` largest entries under (S descending, label ascending): rank(j) = #{k : key_k > key_j,
// or key_k == key_j and k < j} is unique, and j is kept iff rank(j) < keep. Kept labels
// are written in ascending order.
__global__ void __launch_bounds__(kSelWarps * 32) ssba_select_kernel(const float* __restrict__ qb,
                                                                     const float* __restrict__ kb, int Tb,
                                                                     int d, int keep,
                                                                     int32_t* __restrict__ idx,
                                                                     int32_t* __restrict__ cnt,
                                                                     float* __restrict__ scores)
{
    extern __shared__ float sm[];
    constexpr int kLd = kSelKeyChunk + 1;
    float* kbT = sm;
    float* qs = kbT + (size_t)d * kLd;
    uint32_t* Skey = reinterpret_cast<uint32_t*>(qs + (size_t)kSelWarps * d);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int bh = blockIdx.y;
    const int row = blockIdx.x * kSelWarps + warp;
    const bool active = row < Tb;
    const float* kbh = kb + (size_t)bh * Tb * d;
    uint32_t* S = Skey + (size_t)warp * Tb;
    const size_t rowoff = (size_t)bh * Tb + row;

    if (active)
        for (int c = lane; c < d; c += 32) qs[warp * d + c] = qb[rowoff * d + c];

    for (int j0 = 0; j0 < Tb; j0 += kSelKeyChunk) {
        const int nk = min(kSelKeyChunk, Tb - j0);
        __syncthreads();
        // float4 loads (d % 4 == 0), unrolled so that each thread's loads are all in flight
        const float4* src4 = reinterpret_cast<const float4*>(kbh + (size_t)j0 * d);
        const int n4 = nk * d / 4;
#pragma unroll 4
        for (int e4 = threadIdx.x; e4 < n4; e4 += kSelWarps * 32) {
            const float4 v = __ldg(src4 + e4);
            const int e = e4 * 4, j = e / d, c = e - j * d;
            kbT[(c + 0) * kLd + j] = v.x;
            kbT[(c + 1) * kLd + j] = v.y;
            kbT[(c + 2) * kLd + j] = v.z;
            kbT[(c + 3) * kLd + j] = v.w;
        }
        __syncthreads();
        if (active) {
            for (int j = lane; j < nk; j += 32) {
                // four interleaved partial sums over d (c = 4t + u), combined in a fixed order
                float a[4] = {0.f, 0.f, 0.f, 0.f};
                int c = 0;
                for (; c + 4 <= d; c += 4)
#pragma unroll
                    for (int u = 0; u < 4; ++u) a[u] = fmaf(qs[warp * d + c + u], kbT[(c + u) * kLd + j], a[u]);
                for (; c < d; ++c) a[0] = fmaf(qs[warp * d + c], kbT[c * kLd + j], a[0]);
                const float acc = (a[0] + a[1]) + (a[2] + a[3]);
                if (scores) scores[rowoff * Tb + j0 + j] = acc;
                S[j0 + j] = sel::order_key(acc);
            }
        }
    }
    __syncwarp();
    if (!active) return;
    int32_t* dst = idx + rowoff * keep;

    if (Tb <= 32) sel::rank_select<1>(S, Tb, keep, lane, dst);
    else if (Tb <= 64) sel::rank_select<2>(S, Tb, keep, lane, dst);
    else if (Tb <= 128) sel::rank_select<4>(S, Tb, keep, lane, dst);
    else if (Tb <= kRankMaxTb) sel::rank_select<8>(S, Tb, keep, lane, dst);
    else {
        // keep-th largest key by MSB-first radix select
        uint32_t prefix = 0, pmask = 0;
        int remaining = keep;
        for (int bit = 31; bit >= 0; --bit) {
            const uint32_t trial = prefix | (1u << bit), tmask = pmask | (1u << bit);
            int c = 0;
            for (int j = lane; j < Tb; j += 32) c += (S[j] & tmask) == trial;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
            if (c >= remaining) prefix = trial;
            else remaining -= c;
            pmask = tmask;
        }
        // kept: key > T, or key == T among the first `remaining` equal ones (lowest labels)
        const uint32_t T = prefix;
        int out = 0, eq_seen = 0;
        for (int j0 = 0; j0 < Tb; j0 += 32) {
            const int j = j0 + lane;
            const uint32_t key = j < Tb ? S[j] : 0u;
            const bool gt = j < Tb && key > T;
            const bool eq = j < Tb && key == T;
            const uint32_t eqm = __ballot_sync(0xffffffffu, eq);
            const int eq_rank = eq_seen + __popc(eqm & ((1u << lane) - 1u));
            const bool kept = gt || (eq && eq_rank < remaining);
            const uint32_t km = __ballot_sync(0xffffffffu, kept);
            if (kept) dst[out + __popc(km & ((1u << lane) - 1u))] = j;
            out += __popc(km);
            eq_seen += __popc(eqm);
        }
    }
    if (lane == 0) cnt[rowoff] = keep;
}


constexpr int kFuseCluster = 8;    // CTAs per (batch, head)
constexpr int kFuseWarps = 8;
constexpr int kFuseMaxTb = 256;

// Affinity row of one query block (S_j = q_b . k_b[j], four interleaved partial sums over d
// combined in a fixed order, as ssba_select_kernel) with the keys kept in registers (lane l:
// labels l + 32 m), then the radix walk of sel::ballot_select, which keeps the same labels as
// sel::rank_select. kbs: the head's k_b by rows, the 16-byte chunk c4 of row j at chunk
// c4 ^ (j & 15) (the 32 lanes reading one chunk of 32 rows cover all 32 banks: four wavefronts,
// the least for 512 bytes).
template <int kPer>
__device__ __forceinline__ void affinity_select(const float* q, const float* kbs, int Tb, int keep, int lane,
                                                float* srow, int32_t* dst)
{
    constexpr int kD = 64;
    uint32_t key[kPer];
#pragma unroll
    for (int m = 0; m < kPer; ++m) {
        const int j = lane + 32 * m;
        key[m] = 0u;
        if (j < Tb) {
            const float* row = kbs + j * kD;
            const int sw = j & 15;
            float a[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int c = 0; c < kD; c += 4) {
                const float4 qv = *reinterpret_cast<const float4*>(q + c);
                const float4 kv = *reinterpret_cast<const float4*>(row + 4 * ((c >> 2) ^ sw));
                a[0] = fmaf(qv.x, kv.x, a[0]);
                a[1] = fmaf(qv.y, kv.y, a[1]);
                a[2] = fmaf(qv.z, kv.z, a[2]);
                a[3] = fmaf(qv.w, kv.w, a[3]);
            }
            const float acc = (a[0] + a[1]) + (a[2] + a[3]);
            if (srow) srow[j] = acc;
            key[m] = sel::order_key(acc);
        }
    }
    sel::ballot_select<kPer>(key, Tb, keep, lane, dst);
}

// One cluster of kFuseCluster CTAs per (batch*head); CTA r of the cluster owns the blocks
// [r * bpc, (r + 1) * bpc) ∩ [0, Tb).
// smem: qown [bpc][64] | kbs [Tb][64] (the head's k_b, 16-byte chunks swizzled by row)
//   1. pool: warp w takes (block, tensor) units w, w + 8, ... of its CTA; lane l covers
//      16-byte chunk l % CPR of rows l / CPR + RPI * i, summed in row order, then across
//      lanes by shuffles (fixed order); a q_b mean goes to qown, a k_b mean into kbs of every
//      CTA of the cluster (distributed shared memory stores, one per CTA and chunk).
//   2. one cluster barrier (release / acquire: every CTA's stores into kbs are visible after
//      it, and none follow it, so a CTA may leave once it is done).
//   3. one warp per owned query block: S row by four interleaved partial sums over d, its
//      keys in registers, then the radix walk (affinity_select).
template <typename T>
__global__ void __launch_bounds__(kFuseWarps * 32) ssba_mask_fused_kernel(const T* __restrict__ Q,
                                                                          const T* __restrict__ K, Grid g,
                                                                          int keep, int bpc,
                                                                          int32_t* __restrict__ idx,
                                                                          int32_t* __restrict__ cnt,
                                                                          float* __restrict__ scores)
{
    namespace cg = cooperative_groups;
    constexpr int kD = 64;
    constexpr int VE = Vec<T>::kElems;
    constexpr int CPR = kD / VE;      // 16-byte chunks per token row
    constexpr int RPI = 32 / CPR;     // rows per warp instruction
    constexpr int LOADS = 64 / RPI;   // loads per lane per (block, tensor)
    constexpr int BATCH = LOADS < 16 ? LOADS : 16;  // loads in flight per lane
    cg::cluster_group cluster = cg::this_cluster();
    extern __shared__ float smf[];
    const int Tb = g.Tb();
    const int rank = (int)cluster.block_rank();
    const int bh = blockIdx.y;
    const int b0 = rank * bpc;
    const int nb = max(0, min(bpc, Tb - b0));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int N = g.H * g.W;
    float* qown = smf;
    float* kbs = qown + bpc * kD;

    // the k_b stores go into the other CTAs' shared memory, which is only valid once every CTA
    // of the cluster runs: arrive here, wait before the first store (after the first loads)
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    bool started = false;

    // Q and K may come from the grid launched just before this one
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();

    // 1. pool the owned blocks
    const int col = lane % CPR, r0 = lane / CPR;
    for (int u = warp; u < 2 * nb; u += kFuseWarps) {
        const int which = u & 1, k = u >> 1, label = b0 + k;
        const T* X = (which ? K : Q) + (size_t)bh * N * kD + col * VE;
        // window origin in the rolled frame, once per unit; rows and columns of the 8x8
        // window then follow by shifts (the same map as Grid::token with blk = 8)
        const int br = label / g.bw, bc = label - br * g.bw;
        const int rb = br * 8 - g.sr, cb = bc * 8 - g.sc;
        float acc[VE];
#pragma unroll
        for (int e = 0; e < VE; ++e) acc[e] = 0.f;
#pragma unroll
        for (int i0 = 0; i0 < LOADS; i0 += BATCH) {
            uint4 v[BATCH];
#pragma unroll
            for (int i = 0; i < BATCH; ++i) {
                const int pos = r0 + (i0 + i) * RPI;
                int r = rb + (pos >> 3), c = cb + (pos & 7);
                r += r < 0 ? g.H : 0;
                c += c < 0 ? g.W : 0;
                v[i] = __ldg(reinterpret_cast<const uint4*>(X + (size_t)(r * g.W + c) * kD));
            }
#pragma unroll
            for (int i = 0; i < BATCH; ++i) {
                float f[VE];
                Vec<T>::to_f32(v[i], f);
#pragma unroll
                for (int e = 0; e < VE; ++e) acc[e] += f[e];
            }
        }
#pragma unroll
        for (int o = CPR; o < 32; o <<= 1)
#pragma unroll
            for (int e = 0; e < VE; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
        if (!started) {  // warp-uniform
            asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
            started = true;
        }
        if (r0 == 0) {
#pragma unroll
            for (int e = 0; e < VE; ++e) acc[e] *= 1.0f / 64.0f;
            if (!which) {
                float* dst = qown + k * kD + col * VE;
#pragma unroll
                for (int e = 0; e < VE; ++e) dst[e] = acc[e];
            } else {
                // chunks col * VE / 4 .. of row `label`, into the k_b of every CTA of the cluster
#pragma unroll
                for (int r = 0; r < kFuseCluster; ++r) {
                    float* rk = cluster.map_shared_rank(kbs, r) + label * kD;
#pragma unroll
                    for (int h = 0; h < VE / 4; ++h) {
                        const int c4 = col * (VE / 4) + h;
                        *reinterpret_cast<float4*>(rk + 4 * (c4 ^ (label & 15))) =
                            make_float4(acc[4 * h], acc[4 * h + 1], acc[4 * h + 2], acc[4 * h + 3]);
                    }
                }
            }
        }
    }
    if (!started) asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
    // 2. every k_b row of the head is in this CTA's kbs after the barrier
    cluster.sync();

    // 3. affinity rows and selection
    for (int k = warp; k < nb; k += kFuseWarps) {
        const size_t rowoff = (size_t)bh * Tb + b0 + k;
        const float* q = qown + k * kD;
        float* srow = scores ? scores + rowoff * Tb : nullptr;
        int32_t* dst = idx + rowoff * keep;
        if (Tb <= 32) affinity_select<1>(q, kbs, Tb, keep, lane, srow, dst);
        else if (Tb <= 64) affinity_select<2>(q, kbs, Tb, keep, lane, srow, dst);
        else if (Tb <= 128) affinity_select<4>(q, kbs, Tb, keep, lane, srow, dst);
        else affinity_select<8>(q, kbs, Tb, keep, lane, srow, dst);
        if (lane == 0) cnt[rowoff] = keep;
    }
}

// Block means alone, with the pooling loop of ssba_mask_fused_kernel (so the same inputs give
// bit-identical means): CTA = kPoolWin blocks of one (batch*head), warp w pools tensor (w & 1)
// of block w / 2, every load of a lane in flight at once; programmatic dependent launch.
constexpr int kPoolWin = 4;
template <typename T>
__global__ void __launch_bounds__(2 * kPoolWin * 32) ssba_pool_blocks_kernel(const T* __restrict__ Q,
                                                                             const T* __restrict__ K, Grid g,
                                                                             float* __restrict__ qb,
                                                                             float* __restrict__ kb)
{
    constexpr int kD = 64;
    constexpr int VE = Vec<T>::kElems;
    constexpr int CPR = kD / VE;
    constexpr int RPI = 32 / CPR;
    constexpr int LOADS = 64 / RPI;
    constexpr int BATCH = LOADS < 16 ? LOADS : 16;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int Tb = g.Tb();
    const int label = blockIdx.x * kPoolWin + (warp >> 1), which = warp & 1, bh = blockIdx.y;
    const int N = g.H * g.W;
    ptx::grid_dep_wait();
    ptx::grid_dep_launch();
    if (label >= Tb) return;
    const int col = lane % CPR, r0 = lane / CPR;
    const T* X = (which ? K : Q) + (size_t)bh * N * kD + col * VE;
    const int br = label / g.bw, bc = label - br * g.bw;
    const int rb = br * 8 - g.sr, cb = bc * 8 - g.sc;
    float acc[VE];
#pragma unroll
    for (int e = 0; e < VE; ++e) acc[e] = 0.f;
#pragma unroll
    for (int i0 = 0; i0 < LOADS; i0 += BATCH) {
        uint4 v[BATCH];
#pragma unroll
        for (int i = 0; i < BATCH; ++i) {
            const int pos = r0 + (i0 + i) * RPI;
            int r = rb + (pos >> 3), c = cb + (pos & 7);
            r += r < 0 ? g.H : 0;
            c += c < 0 ? g.W : 0;
            v[i] = __ldg(reinterpret_cast<const uint4*>(X + (size_t)(r * g.W + c) * kD));
        }
#pragma unroll
        for (int i = 0; i < BATCH; ++i) {
            float f[VE];
            Vec<T>::to_f32(v[i], f);
#pragma unroll
            for (int e = 0; e < VE; ++e) acc[e] += f[e];
        }
    }
#pragma unroll
    for (int o = CPR; o < 32; o <<= 1)
#pragma unroll
        for (int e = 0; e < VE; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
    if (r0 == 0) {
        float* dst = (which ? kb : qb) + ((size_t)bh * Tb + label) * kD + col * VE;
#pragma unroll
        for (int e = 0; e < VE; ++e) dst[e] = acc[e] * (1.0f / 64.0f);
    }
}

}  // namespace

int launch_pool_blocks(const ssba_desc& d, const Grid& g, const void* Q, const void* K, float* qb, float* kb,
                       cudaStream_t st)
{
    if (d.head_dim != 64 || g.blk != 8) return launch_pool(d, g, Q, K, qb, kb, st);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((g.Tb() + kPoolWin - 1) / kPoolWin, d.B * d.heads, 1);
    cfg.blockDim = dim3(2 * kPoolWin * 32, 1, 1);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e;
    if (d.dtype == SSBA_BF16)
        e = cudaLaunchKernelEx(&cfg, ssba_pool_blocks_kernel<__nv_bfloat16>, static_cast<const __nv_bfloat16*>(Q),
                               static_cast<const __nv_bfloat16*>(K), g, qb, kb);
    else
        e = cudaLaunchKernelEx(&cfg, ssba_pool_blocks_kernel<float>, static_cast<const float*>(Q),
                               static_cast<const float*>(K), g, qb, kb);
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("ssba_pool_blocks_kernel launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

int launch_pool(const ssba_desc& d, const Grid& g, const void* Q, const void* K, float* qb, float* kb,
                cudaStream_t st)
{
    cudaError_t e = cudaSuccess;
    if (d.head_dim == 64 && g.blk == 8) {
        dim3 grid(g.Tb(), d.B * d.heads);
        if (d.dtype == SSBA_BF16)
            ssba_pool_kernel<__nv_bfloat16><<<grid, 256, 0, st>>>(static_cast<const __nv_bfloat16*>(Q),
                                                                  static_cast<const __nv_bfloat16*>(K), g, qb, kb);
        else
            ssba_pool_kernel<float><<<grid, 256, 0, st>>>(static_cast<const float*>(Q), static_cast<const float*>(K),
                                                          g, qb, kb);
        e = cudaGetLastError();
    } else {
        const int P = g.blk * g.blk;
        const size_t smem = (size_t)2 * P * d.head_dim * sizeof(float);
        if (smem > 200 * 1024) {
            set_error("ssba_build_mask: block*block*head_dim too large for the pooling kernel");
            return SSBA_ERR_UNSUPPORTED;
        }
        dim3 grid(g.Tb(), d.B * d.heads);
        if (d.dtype == SSBA_BF16) {
            auto k = ssba_pool_generic_kernel<__nv_bfloat16>;
            if (smem > 48 * 1024) cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            k<<<grid, 128, smem, st>>>(static_cast<const __nv_bfloat16*>(Q), static_cast<const __nv_bfloat16*>(K), g,
                                       d.head_dim, qb, kb);
        } else {
            auto k = ssba_pool_generic_kernel<float>;
            if (smem > 48 * 1024) cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            k<<<grid, 128, smem, st>>>(static_cast<const float*>(Q), static_cast<const float*>(K), g, d.head_dim, qb,
                                       kb);
        }
        e = cudaGetLastError();
    }
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
    size_t smem = ((size_t)d.head_dim * (kSelKeyChunk + 1) + (size_t)kSelWarps * d.head_dim +
                   (size_t)kSelWarps * Tb) * sizeof(float);
    if (smem > 220 * 1024) {
        set_error("ssba_build_mask: selection working set too large (%zu bytes)", smem);
        return SSBA_ERR_UNSUPPORTED;
    }
    cudaFuncSetAttribute(ssba_select_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                         cudaSharedmemCarveoutMaxShared);
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

namespace ssba {

// The fused mask build (one launch) when the shape allows it; returns SSBA_ERR_UNSUPPORTED
// (without launching and without setting an error) otherwise.
int launch_mask_fused(const ssba_desc& d, const Grid& g, int keep, const void* Q, const void* K, int32_t* idx,
                      int32_t* cnt, float* scores, cudaStream_t st)
{
    const int Tb = g.Tb();
    if (d.head_dim != 64 || g.blk != 8 || Tb > kFuseMaxTb) return SSBA_ERR_UNSUPPORTED;
    const int bpc = (Tb + kFuseCluster - 1) / kFuseCluster;
    const size_t smem = ((size_t)bpc * 64 + (size_t)Tb * 64) * sizeof(float);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kFuseCluster, d.B * d.heads, 1);
    cfg.blockDim = dim3(kFuseWarps * 32, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kFuseCluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see grid_dep_wait
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    cudaError_t e;
    if (d.dtype == SSBA_BF16) {
        auto k = ssba_mask_fused_kernel<__nv_bfloat16>;
        if (smem > 48 * 1024) cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        e = cudaLaunchKernelEx(&cfg, k, static_cast<const __nv_bfloat16*>(Q), static_cast<const __nv_bfloat16*>(K),
                               g, keep, bpc, idx, cnt, scores);
    } else {
        auto k = ssba_mask_fused_kernel<float>;
        if (smem > 48 * 1024) cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        e = cudaLaunchKernelEx(&cfg, k, static_cast<const float*>(Q), static_cast<const float*>(K), g, keep, bpc, idx,
                               cnt, scores);
    }
    if (e != cudaSuccess) {
        set_error("ssba_mask_fused_kernel launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

}  // namespace ssba
