// qkv.cu -- the steps of Algorithm 1 before the mask, fused into one tensor-core GEMM:
// the QKV projection of the image tokens, RoPE on Q and K (first step of Algorithm 1, read
// as 2-D axial RoPE), and the block compression of Sec. 2.2 (mean of Q and of K over each
// 8x8 window of the layer's shifted grid), so that the mask build no longer re-reads Q and K.
//
//   Y = X Wqkv^T + bias        X [B][N][Dm] bf16 (tokens in grid order), Wqkv [3 Dm][Dm] bf16
//   Q, K = RoPE(Y_q), RoPE(Y_k), V = Y_v, each [B][heads][N][64] bf16
//   q_b, k_b = block means of the bf16 Q and K, [B][heads][Tb][64] fp32
//
// Tile = 128 rows (two horizontally adjacent 8x8 windows of the shifted grid, one 16 x 8
// token box per k step, so that the rows of a tile come from long runs of consecutive tokens:
// measured, two 8 x 8 boxes per k step took the main loop from 35 to 47 us at 1024 px) x 256
// output columns (four heads of 64) x the whole Dm, in 64-wide k steps through a 4-stage ring
// of 48 KB (A 16 KB + B 32 KB, 128-byte swizzle). A pair that crosses the grid edge (shifted
// layers) is cut into two or four boxes of 4, 8 or 12 columns and 4 or 8 rows. Persistent
// CTAs, one per SM, 320 threads:
//   warp 0      TMA producer (one elected lane)
//   warp 1      MMA issuer: tcgen05.mma kind::f16 M=128 N=256 K=16, four per k step, into one
//               of two 256-column TMEM accumulators (512 columns), so that the epilogue of
//               tile i overlaps the main loop of tile i+1; also owns the TMEM allocation
//   warps 2-9   epilogue, two warps per TMEM lane quadrant (row = lane), each taking two of
//               the tile's four heads in 32-column chunks: bias, RoPE in fp32 with cos/sin
//               from a per-CTA table, bf16 stores of 64 bytes per token and chunk, and the
//               window sums of the rounded Q and K. In a tile of one 16 x 8 box, bit 3 of the
//               lane is the window, and a four-step butterfly leaves each lane the sums of two
//               columns of its window over the quadrant's rows; other tiles take a masked
//               five-step butterfly per window. The four quadrants' sums meet in shared
//               memory (mbarriers with bounded waits) and one warp adds them in a fixed order
//               and writes the means (no atomics).
// All mbarrier waits are bounded (globaltimer budget + CTA abort flag); a timeout is written
// to the device status word and the CTA drains its in-flight copies and MMAs before exiting.
#include <cuda.h>
#include <cstddef>
#include <cstring>

#include "common.cuh"
#include "ptx.cuh"

namespace ssba {

namespace {

using namespace ptx;

constexpr int kD = 64;
constexpr int kBM = 128;  // rows of a tile: two windows
constexpr int kBN = 256;  // columns of a tile: four heads
constexpr int kBK = 64;   // k per stage (one 128-byte swizzle atom of bf16)
constexpr int kStages = 4;
constexpr uint32_t kABytes = kBM * kBK * 2;   // 16 KB
constexpr uint32_t kBBytes = kBN * kBK * 2;   // 32 KB
constexpr uint32_t kIdesc = idesc_bf16_f32(kBM, kBN, false, false);
constexpr int kEpiWarps = 8;
constexpr int kThreads = (2 + kEpiWarps) * 32;
constexpr uint32_t kTmemCols = 2 * kBN;
constexpr int kNumFreq = kD / 4;  // RoPE frequencies per axis
constexpr int kRopeCap = 128;     // grid rows / columns whose cos, sin are tabulated per CTA

struct QkvMaps {
    CUtensorMap x[8];  // X as [B*H][W][Dm]: boxes of 4, 8, 12, 16 columns x 8 rows, then x 4 rows
    CUtensorMap w;     // Wqkv as [1][3 Dm][Dm], 256-row boxes
};

__device__ __forceinline__ const CUtensorMap* xbox(const QkvMaps& m, int cols, int rows)
{
    return &m.x[(cols >> 2) - 1 + (rows == 4 ? 4 : 0)];
}

struct QkvParams {
    __nv_bfloat16* q;
    __nv_bfloat16* k;
    __nv_bfloat16* v;
    float* qb;  // null: no pooling
    float* kb;
    const float* bias;  // null: none
    Grid g;
    int B, heads, Dm;
    int pairs;  // window pairs per window row: ceil(W / 16)
    int m_tiles, n_tiles, tiles;
    float theta[kNumFreq];
    int* status;
    uint64_t budget_ns;
};

struct __align__(1024) QkvSmem {
    uint8_t a[kStages][kABytes];
    uint8_t b[kStages][kBBytes];
    uint64_t full[kStages], empty[kStages];
    uint64_t acc_full[2], acc_empty[2];
    uint64_t drain;
    uint64_t pool_full[2], pool_free[2];  // per head pair: the quadrants' sums written / taken
    uint64_t bias_full[2];                // per accumulator: the tile's bias has landed
    alignas(16) float bias[2][kBN];       // per accumulator: the tile's 256 biases (bulk-copy target)
    float part[2][4][2][2][2][32];        // [head pair][quadrant][head][chunk][window][column]
    float2 rope[kNumFreq][kRopeCap];  // (cos, sin) of pos * theta_i
    uint32_t tmem_base;
    int abort_flag;
};

// every TMA / bulk-copy destination starts on the alignment its copy needs
static_assert(offsetof(QkvSmem, a) % 1024 == 0 && offsetof(QkvSmem, b) % 1024 == 0, "stage alignment");
static_assert(kABytes % 1024 == 0 && kBBytes % 1024 == 0, "stage size");
static_assert(offsetof(QkvSmem, bias) % 16 == 0 && (kBN * sizeof(float)) % 16 == 0, "bias alignment");

// A tile's rows: the pair of windows (window row wr, windows 2 pp and 2 pp + 1) of one image,
// a 16 x 8 region of the rolled grid (8 x 8 when the row has an odd last window). Its origin
// in the unshifted grid is (r0, c0); w1 > 0 when the region crosses the right edge (the first
// w1 columns, then the rest from column 0), rs when it crosses the bottom edge (4 + 4 rows).
struct TileGeo {
    int b, nt, L0, wd, r0, c0, w1;
    bool rs, two;
};

__device__ __forceinline__ TileGeo tile_geo(const QkvParams& p, const Grid& g, int t)
{
    TileGeo o;
    o.nt = t % p.n_tiles;
    const int rest = t / p.n_tiles;
    const int mt = rest % p.m_tiles;
    o.b = rest / p.m_tiles;
    const int wr = mt / p.pairs, pp = mt - wr * p.pairs;
    o.L0 = wr * g.bw + 2 * pp;
    o.two = 2 * pp + 1 < g.bw;
    o.wd = o.two ? 16 : 8;
    o.r0 = wr * 8 - g.sr;
    if (o.r0 < 0) o.r0 += g.H;
    o.c0 = 16 * pp - g.sc;
    if (o.c0 < 0) o.c0 += g.W;
    o.rs = o.r0 + 8 > g.H;
    o.w1 = o.c0 + o.wd > g.W ? g.W - o.c0 : 0;
    return o;
}

// The region's rows of k step k0 into dst (rows in box order, 128 bytes each).
__device__ __forceinline__ void load_tile(const QkvMaps& m, uint32_t dst, uint32_t bar, const Grid& g,
                                          const TileGeo& o, int k0)
{
    const int row0 = o.b * g.H, wd = o.wd, w1 = o.w1, w2 = wd - w1;
    if (!w1 && !o.rs) {
        tma_load_3d(dst, xbox(m, wd, 8), bar, k0, o.c0, row0 + o.r0);
    } else if (!w1) {
        tma_load_3d(dst, xbox(m, wd, 4), bar, k0, o.c0, row0 + o.r0);
        tma_load_3d(dst + 4 * wd * 128, xbox(m, wd, 4), bar, k0, o.c0, row0);
    } else if (!o.rs) {
        tma_load_3d(dst, xbox(m, w1, 8), bar, k0, o.c0, row0 + o.r0);
        tma_load_3d(dst + 8 * w1 * 128, xbox(m, w2, 8), bar, k0, 0, row0 + o.r0);
    } else {
        tma_load_3d(dst, xbox(m, w1, 4), bar, k0, o.c0, row0 + o.r0);
        tma_load_3d(dst + 4 * w1 * 128, xbox(m, w2, 4), bar, k0, 0, row0 + o.r0);
        tma_load_3d(dst + 4 * wd * 128, xbox(m, w1, 4), bar, k0, o.c0, row0);
        tma_load_3d(dst + 4 * wd * 128 + 4 * w1 * 128, xbox(m, w2, 4), bar, k0, 0, row0);
    }
}

// Tile row rho (< 8 wd) -> (row a, column c) of the region, following the box order of load_tile.
__device__ __forceinline__ void tile_rc(const TileGeo& o, int rho, int& a, int& c)
{
    const int wd = o.wd, w1 = o.w1, w2 = wd - w1;
    if (!w1) {  // one box, or two row halves
        a = rho / wd;
        c = rho - a * wd;
    } else if (!o.rs) {  // two column parts
        if (rho < 8 * w1) {
            a = rho / w1;
            c = rho - a * w1;
        } else {
            const int q = rho - 8 * w1;
            a = q / w2;
            c = w1 + q - (q / w2) * w2;
        }
    } else {  // four parts: top-left, top-right, bottom-left, bottom-right
        const int h = rho / (4 * wd), q0 = rho - h * 4 * wd;
        if (q0 < 4 * w1) {
            a = 4 * h + q0 / w1;
            c = q0 - (q0 / w1) * w1;
        } else {
            const int q = q0 - 4 * w1;
            a = 4 * h + q / w2;
            c = w1 + q - (q / w2) * w2;
        }
    }
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float2 unpack2(uint32_t w) { return __bfloat1622float2(*reinterpret_cast<__nv_bfloat162*>(&w)); }

__device__ __forceinline__ bool wait_raw_q(uint32_t bar, uint32_t parity, uint64_t budget_ns)
{
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity))
        if (globaltimer_ns() - t0 > budget_ns) return false;
    return true;
}

// kTable: RoPE cos/sin from the per-CTA table (grids up to kRopeCap rows and columns); else
// computed per element (a separate instantiation, so that the table path stays compact).
template <bool kTable>
__global__ void __launch_bounds__(kThreads, 1) ssba_qkv_rope_pool_kernel(const __grid_constant__ QkvMaps maps,
                                                                          const QkvParams p)
{
    extern __shared__ uint8_t smem_raw[];
    QkvSmem& sm = *reinterpret_cast<QkvSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abortf = &sm.abort_flag;
    const Grid g = p.g;
    const int Tb = g.Tb();
    const int N = g.H * g.W;
    const int ksteps = p.Dm / kBK;

    if (threadIdx.x == 0) {
        sm.abort_flag = 0;
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&sm.full[s]), 1);
            mbar_init(smem_u32(&sm.empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&sm.acc_full[b]), 1);
            mbar_init(smem_u32(&sm.acc_empty[b]), kEpiWarps);
        }
        mbar_init(smem_u32(&sm.drain), 1);
        for (int hp = 0; hp < 2; ++hp) {
            mbar_init(smem_u32(&sm.pool_full[hp]), 4);
            mbar_init(smem_u32(&sm.pool_free[hp]), 1);
            mbar_init(smem_u32(&sm.bias_full[hp]), 1);
        }
        fence_mbar_init();
    }
    if (warp == 0 && lane < 9) tma_prefetch_desc(lane < 8 ? &maps.x[lane] : &maps.w);
    if constexpr (kTable) {
        const int npos = max(g.H, g.W);
        for (int e = threadIdx.x; e < kNumFreq * npos; e += kThreads) {
            const int i = e / npos, pos = e - i * npos;
            float sv, cv;
            sincosf((float)pos * p.theta[i], &sv, &cv);
            sm.rope[i][pos] = make_float2(cv, sv);
        }
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = sm.tmem_base;
    bool dead = false;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        uint32_t gstep = 0;
        if (lane == 0) {
            for (int t = blockIdx.x; t < p.tiles && !dead; t += gridDim.x) {
                const TileGeo o = tile_geo(p, g, t);
                for (int ks = 0; ks < ksteps; ++ks, ++gstep) {
                    const uint32_t s = gstep % kStages;
                    if (!mbar_wait(smem_u32(&sm.empty[s]), ((gstep / kStages) & 1) ^ 1, abortf, p.budget_ns)) {
                        dead = true;
                        break;
                    }
                    const uint32_t bar = smem_u32(&sm.full[s]);
                    mbar_arrive_expect_tx(bar, 8 * o.wd * 128 + kBBytes);
                    load_tile(maps, smem_u32(&sm.a[s][0]), bar, g, o, ks * kBK);
                    tma_load_3d(smem_u32(&sm.b[s][0]), &maps.w, bar, ks * kBK, o.nt * kBN, 0);
                }
            }
            if (dead) {
                // drain: the copies of the last stages issued may still be in flight
                for (uint32_t x = gstep > kStages ? gstep - kStages : 0; x < gstep; ++x)
                    wait_raw_q(smem_u32(&sm.full[x % kStages]), (x / kStages) & 1, p.budget_ns);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        const bool leader = elect_one_sync();
        uint32_t gstep = 0, it = 0, nbias = 0;
        const uint32_t a0 = smem_u32(&sm.a[0][0]), b0 = smem_u32(&sm.b[0][0]);
        for (int t = blockIdx.x; t < p.tiles && !dead; t += gridDim.x, ++it) {
            const uint32_t acc = it & 1;
            if (!mbar_wait(smem_u32(&sm.acc_empty[acc]), ((it >> 1) & 1) ^ 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            tc_fence_after();
            if (p.bias && lane == 0) {
                // the tile's biases, for the epilogue, into the buffer of this accumulator
                const int c0 = (t % p.n_tiles) * kBN;
                const uint32_t bytes = (uint32_t)min(kBN, 3 * p.Dm - c0) * 4;
                mbar_arrive_expect_tx(smem_u32(&sm.bias_full[acc]), bytes);
                bulk_load(smem_u32(&sm.bias[acc][0]), p.bias + c0, bytes, smem_u32(&sm.bias_full[acc]));
                ++nbias;
            }
            __syncwarp();
            const uint32_t d = tbase + acc * kBN;
            for (int ks = 0; ks < ksteps; ++ks, ++gstep) {
                const uint32_t s = gstep % kStages;
                if (!mbar_wait(smem_u32(&sm.full[s]), (gstep / kStages) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                if (leader) {
                    const uint64_t ad = sdesc_sw128(a0 + s * kABytes, 16, 1024);
                    const uint64_t bd = sdesc_sw128(b0 + s * kBBytes, 16, 1024);
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k)
                        mma_ss(d, ad + (uint64_t)(k * 2), bd + (uint64_t)(k * 2), kIdesc, (ks | k) != 0 ? 1u : 0u);
                    mma_commit(smem_u32(&sm.empty[s]));
                    if (ks == ksteps - 1) mma_commit(smem_u32(&sm.acc_full[acc]));
                }
                __syncwarp();
            }
        }
        if (dead && leader) {
            mma_commit(smem_u32(&sm.drain));
            wait_raw_q(smem_u32(&sm.drain), 0, p.budget_ns);
        }
        if (dead && lane == 0 && nbias > 0) {
            // the last bias copy issued may still be in flight
            const uint32_t last = nbias - 1;  // every tile issues one copy: this is its tile count
            wait_raw_q(smem_u32(&sm.bias_full[last & 1]), (last >> 1) & 1, p.budget_ns);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        const int quad = warp & 3;          // TMEM lanes [32 quad, 32 quad + 32)
        const int hp = (warp - 2) >> 2;    // heads 2 hp and 2 hp + 1 of the tile
        const int rho = 32 * quad + lane;  // tile row
        const bool collector = quad == 0;  // adds the four quadrants' sums and writes the means
        uint32_t it = 0, npool = 0;
        for (int t = blockIdx.x; t < p.tiles && !dead; t += gridDim.x, ++it) {
            const TileGeo o = tile_geo(p, g, t);
            int ra, rc;
            tile_rc(o, rho, ra, rc);
            const int win = rc >> 3;
            const bool valid = rho < 8 * o.wd;
            const int tok = valid ? g.token(o.L0 + win, ra * 8 + (rc & 7)) : 0;
            const int tpos[2] = {tok / g.W, tok % g.W};  // RoPE positions: row, column
            // stores go out transposed within groups of four lanes (see below): the tokens and
            // validity of the group's rows
            int tokm[4];
            bool validm[4];
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                tokm[m] = __shfl_sync(0xffffffffu, tok, (lane & ~3) | m);
                validm[m] = __shfl_sync(0xffffffffu, (int)valid, (lane & ~3) | m) != 0;
            }
            const bool regular = o.wd == 16 && o.w1 == 0;  // window = bit 3 of the lane
            const int b = o.b, nt = o.nt;
            const uint32_t acc = it & 1;
            if (!mbar_wait(smem_u32(&sm.acc_full[acc]), (it >> 1) & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            tc_fence_after();
            if (p.bias && !mbar_wait(smem_u32(&sm.bias_full[acc]), (it >> 1) & 1, abortf, p.budget_ns)) dead = true;
            const float* bias_t = sm.bias[acc];
            // the warp's heads pool when they hold Q or K (the same for the four quadrants of a
            // head pair, so that their handshake counts agree)
            const int col0 = nt * kBN + hp * 2 * kD;
            const bool pool_tile = col0 < 2 * p.Dm && p.qb != nullptr;
            float(*mypart)[2][2][32] = sm.part[hp][quad];
            if (pool_tile && !collector) {
                // the collector must have taken the previous tile's sums
                if (!mbar_wait(smem_u32(&sm.pool_free[hp]), (npool & 1) ^ 1, abortf, p.budget_ns)) dead = true;
            }
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const int col = col0 + hh * kD;  // first output column of this head
                if (dead || col >= 3 * p.Dm) continue;
                const int which = col / p.Dm, head = (col - which * p.Dm) / kD;
                __nv_bfloat16* outp = which == 0 ? p.q : (which == 1 ? p.k : p.v);
                __nv_bfloat16* headp = outp + ((size_t)b * p.heads + head) * N * kD;
                // both chunks of the head from TMEM behind one wait
                uint32_t rr[2][32];
                {
                    const uint32_t taddr = tbase + ((uint32_t)(32 * quad) << 16) + acc * kBN + (col - nt * kBN);
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        tmem_ld_32x32b_x16(taddr + 16 * j, *reinterpret_cast<uint32_t(*)[16]>(&rr[j >> 1][16 * (j & 1)]));
                    tmem_wait_ld();
                }
#pragma unroll
                for (int ch = 0; ch < 2; ++ch) {  // chunk 0: dims [0, 32) turn with the row, chunk 1 with the column
                    const uint32_t(&r)[32] = rr[ch];
                    float2 cs[kNumFreq];
                    if (which < 2) {
                        const int pos = tpos[ch];
#pragma unroll
                        for (int i = 0; i < kNumFreq; ++i) {
                            if constexpr (kTable)
                                cs[i] = sm.rope[i][pos];
                            else
                                sincosf((float)pos * p.theta[i], &cs[i].y, &cs[i].x);
                        }
                    }
                    float4 bb[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        bb[e] = p.bias ? reinterpret_cast<const float4*>(bias_t + (col - nt * kBN) + 32 * ch)[e]
                                       : make_float4(0.f, 0.f, 0.f, 0.f);
                    float v[32];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        v[4 * e] = __uint_as_float(r[4 * e]) + bb[e].x;
                        v[4 * e + 1] = __uint_as_float(r[4 * e + 1]) + bb[e].y;
                        v[4 * e + 2] = __uint_as_float(r[4 * e + 2]) + bb[e].z;
                        v[4 * e + 3] = __uint_as_float(r[4 * e + 3]) + bb[e].w;
                    }
                    if (which < 2) {
#pragma unroll
                        for (int i = 0; i < kNumFreq; ++i) {
                            const float x0 = v[2 * i], x1 = v[2 * i + 1];
                            v[2 * i] = x0 * cs[i].x - x1 * cs[i].y;
                            v[2 * i + 1] = x0 * cs[i].y + x1 * cs[i].x;
                        }
                    }
                    uint32_t o[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) o[i] = pack2(v[2 * i], v[2 * i + 1]);
                    {
                        // 4 x 4 transpose of 16-byte pieces within each group of four lanes, so
                        // that store m writes 64 contiguous bytes of row (group + m) from four
                        // lanes: 8 lines per store instead of 32 (measured: the 32-line stores
                        // held the next chunk's shared-memory loads for ~2800 cycles)
                        uint4 X[4];
#pragma unroll
                        for (int i = 0; i < 4; ++i) X[i] = make_uint4(o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
                        const int k4 = lane & 3;
#pragma unroll
                        for (int stage = 0; stage < 2; ++stage) {
                            const int bit = 1 << stage;
                            const bool hi = k4 & bit;
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                if (q & bit) continue;  // slot pairs (q, q + bit)
                                const uint4 send = hi ? X[q] : X[q + bit];
                                uint4 recv;
                                recv.x = __shfl_xor_sync(0xffffffffu, send.x, bit);
                                recv.y = __shfl_xor_sync(0xffffffffu, send.y, bit);
                                recv.z = __shfl_xor_sync(0xffffffffu, send.z, bit);
                                recv.w = __shfl_xor_sync(0xffffffffu, send.w, bit);
                                if (hi)
                                    X[q] = recv;
                                else
                                    X[q + bit] = recv;
                            }
                        }
                        // X[m] = piece k4 of row (group + m)
#pragma unroll
                        for (int m = 0; m < 4; ++m)
                            if (validm[m])
                                *reinterpret_cast<uint4*>(headp + (size_t)tokm[m] * kD + 32 * ch + 8 * k4) = X[m];
                    }
                    if (pool_tile && which < 2) {
                        // column sums of the rounded values over the quadrant's rows, per window
                        float a[32];
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const float2 f = unpack2(o[i]);
                            a[2 * i] = valid ? f.x : 0.f;
                            a[2 * i + 1] = valid ? f.y : 0.f;
                        }
                        if (regular) {
                            // lanes l and l ^ 8 hold the two windows: reduce over lane bits 4, 2,
                            // 1, 0; lane l ends with columns base, base + 1 of its window
#pragma unroll
                            for (int k = 0, width = 16; k < 4; ++k, width >>= 1) {
                                const int bit = k == 0 ? 16 : (4 >> (k - 1));
                                const bool up = lane & bit;
#pragma unroll
                                for (int j = 0; j < width; ++j) {
                                    const float send = up ? a[j] : a[j + width];
                                    const float keep = up ? a[j + width] : a[j];
                                    a[j] = keep + __shfl_xor_sync(0xffffffffu, send, bit);
                                }
                            }
                            const int base = ((lane >> 4) & 1) * 16 + ((lane >> 2) & 1) * 8 + ((lane >> 1) & 1) * 4 +
                                             (lane & 1) * 2;
                            mypart[hh][ch][win][base] = a[0];
                            mypart[hh][ch][win][base + 1] = a[1];
                        } else {
                            // masked per window, full five-step butterfly: lane l ends with column l
#pragma unroll
                            for (int w = 0; w < 2; ++w) {
                                float m[32];
#pragma unroll
                                for (int j = 0; j < 32; ++j) m[j] = win == w ? a[j] : 0.f;
#pragma unroll
                                for (int width = 16; width >= 1; width >>= 1) {
                                    const bool up = lane & width;
#pragma unroll
                                    for (int j = 0; j < width; ++j) {
                                        const float send = up ? m[j] : m[j + width];
                                        const float keep = up ? m[j + width] : m[j];
                                        m[j] = keep + __shfl_xor_sync(0xffffffffu, send, width);
                                    }
                                }
                                mypart[hh][ch][w][lane] = m[0];
                            }
                        }
                    }
                }
            }
            if (pool_tile && !dead) {
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&sm.pool_full[hp]));
                if (collector) {
                    if (mbar_wait(smem_u32(&sm.pool_full[hp]), npool & 1, abortf, p.budget_ns)) {
#pragma unroll
                        for (int hh = 0; hh < 2; ++hh) {
                            const int col = col0 + hh * kD;
                            if (col >= 2 * p.Dm) continue;
                            const int which = col / p.Dm, head = (col - which * p.Dm) / kD;
                            float* base = (which == 0 ? p.qb : p.kb) + ((size_t)b * p.heads + head) * Tb * kD;
#pragma unroll
                            for (int w = 0; w < 2; ++w) {
                                if (w == 1 && !o.two) continue;
                                float* dstp = base + (size_t)(o.L0 + w) * kD;
#pragma unroll
                                for (int ch = 0; ch < 2; ++ch) {
                                    float sum = sm.part[hp][0][hh][ch][w][lane];
                                    sum += sm.part[hp][1][hh][ch][w][lane];
                                    sum += sm.part[hp][2][hh][ch][w][lane];
                                    sum += sm.part[hp][3][hh][ch][w][lane];
                                    dstp[32 * ch + lane] = sum * (1.0f / 64.0f);
                                }
                            }
                        }
                        __syncwarp();
                        if (lane == 0) mbar_arrive(smem_u32(&sm.pool_free[hp]));
                    } else {
                        dead = true;
                    }
                }
            }
            if (pool_tile) ++npool;
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&sm.acc_empty[acc]));
        }
    }

    if (dead) atomicExch(p.status, SSBA_ERR_TIMEOUT);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tbase, kTmemCols);
}

bool encode_maps(QkvMaps& m, const void* X, const void* Wqkv, int B, int H, int W, int Dm)
{
    EncodeTiledFn fn = tensor_map_encoder();
    if (!fn) return false;
    for (int s = 0; s < 8; ++s) {
        cuuint64_t dims[3] = {(cuuint64_t)Dm, (cuuint64_t)W, (cuuint64_t)H * B};
        cuuint64_t strides[2] = {(cuuint64_t)Dm * 2, (cuuint64_t)W * Dm * 2};
        cuuint32_t box[3] = {kBK, (cuuint32_t)(4 * (s % 4) + 4), s < 4 ? 8u : 4u};
        cuuint32_t es[3] = {1, 1, 1};
        if (fn(&m.x[s], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(X), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return false;
    }
    cuuint64_t dims[3] = {(cuuint64_t)Dm, (cuuint64_t)3 * Dm, 1};
    cuuint64_t strides[2] = {(cuuint64_t)Dm * 2, (cuuint64_t)3 * Dm * Dm * 2};
    cuuint32_t box[3] = {kBK, kBN, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return fn(&m.w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(Wqkv), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() { return device_sm_count(); }

}  // namespace

int launch_qkv_rope_pool(const ssba_desc& d, const Grid& g, const void* X, const void* Wqkv, const float* bias,
                         void* Q, void* K, void* V, float* qb, float* kb, cudaStream_t st, uint64_t budget_ns)
{
    if (d.head_dim != kD || g.blk != 8 || (g.sr % 4) || (g.sc % 4) || d.dtype != SSBA_BF16) {
        set_error("ssba_qkv_rope_pool: needs bf16, head_dim=64, block=8 and shifts that are multiples of 4");
        return SSBA_ERR_UNSUPPORTED;
    }
    if (g.H >= 32768 || g.W >= 32768) {
        set_error("ssba_qkv_rope_pool: H_tok and W_tok must be below 32768");
        return SSBA_ERR_UNSUPPORTED;
    }
    const int Dm = d.heads * kD;
    QkvMaps maps;
    memset(&maps, 0, sizeof(maps));
    if (!encode_maps(maps, X, Wqkv, d.B, g.H, g.W, Dm)) {
        set_error("ssba_qkv_rope_pool: cuTensorMapEncodeTiled failed");
        return SSBA_ERR_CUDA;
    }
    QkvParams p;
    memset(&p, 0, sizeof(p));
    p.q = static_cast<__nv_bfloat16*>(Q);
    p.k = static_cast<__nv_bfloat16*>(K);
    p.v = static_cast<__nv_bfloat16*>(V);
    p.qb = qb;
    p.kb = kb;
    p.bias = bias;
    p.g = g;
    p.B = d.B;
    p.heads = d.heads;
    p.Dm = Dm;
    p.pairs = (g.bw + 1) / 2;
    p.m_tiles = (g.H / 8) * p.pairs;
    p.n_tiles = (3 * Dm + kBN - 1) / kBN;
    p.tiles = d.B * p.m_tiles * p.n_tiles;
    for (int i = 0; i < kNumFreq; ++i) p.theta[i] = (float)pow(10000.0, -(double)i / kNumFreq);
    p.budget_ns = budget_ns;
    p.status = device_status_word();
    if (!p.status) {
        set_error("ssba_qkv_rope_pool: could not resolve the device status word");
        return SSBA_ERR_CUDA;
    }
    const size_t smem = sizeof(QkvSmem) + 1024;
    static PerDeviceOnce attr;  // shared-memory attributes, set once per device
    attr.run([smem] {
        cudaFuncSetAttribute(ssba_qkv_rope_pool_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        cudaFuncSetAttribute(ssba_qkv_rope_pool_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    });
    const int grid = p.tiles < sm_count() ? p.tiles : sm_count();
    if (g.H <= kRopeCap && g.W <= kRopeCap)
        ssba_qkv_rope_pool_kernel<true><<<grid, kThreads, smem, st>>>(maps, p);
    else
        ssba_qkv_rope_pool_kernel<false><<<grid, kThreads, smem, st>>>(maps, p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("ssba_qkv_rope_pool_kernel launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

}  // namespace ssba
