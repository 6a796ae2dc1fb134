// attn_dense.cu -- dense bf16 softmax attention on the sm_103a tensor cores: the 0 % sparsity
// baseline of Table 2 (every key of the head), the denominator of the sparse kernel's speed-up.
//
// Without index lists every query shares every key, so tiles are 128 contiguous tokens and the
// products run at M=128 (the sparse kernel's 64-row tiles are forced by its per-query-block
// lists, and M=64 products run at half the per-SM rate):
//   S = Q_u K_j^T   tcgen05.mma kind::f16, M=128 N=128 K=16 x 4 (A = Q tile, B = K tile, both
//                   K-major SW128 in shared memory)
//   O += P V_j      M=128 N=64 K=16 x 8 (A = P, bf16, from tensor memory; B = V tile MN-major)
// Work unit = one tile of 128 query rows of one (batch, head); it visits all N/128 key tiles.
// Persistent CTAs, one per SM (their shared memory fills it), each running two independent
// streams of units (unit v + r V for stream v of V), warp-specialised:
//   warps 0, 1     TMA producers of stream 0, 1: the unit's Q tile (double-buffered), then K_j and
//                  V_j into 2-stage rings (16 KB tiles, 128-row boxes of a [B*heads][N][64] map)
//   warps 2, 3     MMA issuers of stream 0, 1 (one elected lane): QK_j once the softmax has
//                  loaded S_{j-1}, then PV_{j-1} once its P is stored, so the tensor pipe has the
//                  next QK while the softmax works
//   warps 4-7      softmax of stream 0, warps 8-11 of stream 1: one thread per row (TMEM lane),
//                  128 scores a tile read in four 32-column chunks twice (maximum, then exp2s and
//                  the bf16 P store), lazy rescale of O by more than 2^8 as in the sparse kernel
//   warps 12-15    epilogue of stream 0, warps 16-19 of stream 1: O / l in bf16 and lse
// TMEM of a stream: S 128 + P 64 (bf16 pairs) + O 64 = 256 columns; the two streams take 512.
// Every mbarrier wait is bounded (globaltimer budget + CTA abort flag); a timeout is reported in
// the device status word and the roles drain their copies and products before the CTA exits.
#include <cuda.h>
#include <cstring>

#include "common.cuh"
#include "ptx.cuh"

namespace ssba {
namespace {

using namespace ptx;

constexpr int kD = 64;
constexpr int kTile = 128;                        // query rows of a unit = keys of a key tile
constexpr uint32_t kTileBytes = kTile * kD * 2;   // 16 KB
constexpr int kStages = 2;                        // K and V rings
constexpr int kStreams = 2;
constexpr int kWarps = 20;
constexpr int kThreads = kWarps * 32;
constexpr uint32_t kStreamCols = 256;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;    // [0,128)
constexpr uint32_t kColP = 128;  // [128,192)
constexpr uint32_t kColO = 192;  // [192,256)
constexpr float kRescaleLog2 = 8.0f;
constexpr uint32_t kIdescQK = idesc_bf16_f32(128, 128, false, false);
constexpr uint32_t kIdescPV = idesc_bf16_f32(128, 64, false, true);

struct __align__(1024) StreamSmem {
    uint8_t q[2][kTileBytes];
    uint8_t k[kStages][kTileBytes];
    uint8_t v[kStages][kTileBytes];
    float2 stats[2][kTile];  // (max in log2 units, row sum) per unit parity
    uint64_t q_full[2], q_empty[2];
    uint64_t k_full[kStages], k_empty[kStages];
    uint64_t v_full[kStages], v_empty[kStages];
    uint64_t s_full, s_free, p_full, p_empty;
    uint64_t stats_full[2], stats_free[2];
    uint64_t o_full, o_free;
    uint64_t drain[2];
};

struct __align__(1024) DenseSmem {
    StreamSmem st[kStreams];
    uint32_t tmem_base;
    int abort_flag;
};
static_assert(sizeof(DenseSmem) + 1024 <= 232448, "shared memory of one CTA (227 KB opt-in limit)");

struct DenseParams {
    __nv_bfloat16* O;
    float* lse;
    int BH;           // batch * heads
    int N;            // tokens, a multiple of 128
    int nt;           // N / 128 tiles a head
    int units;        // BH * nt
    float scale_log2; // softmax scale * log2(e)
    int* status;
    uint64_t budget_ns;
};

struct DenseMaps {
    CUtensorMap q, k, v;
};

__device__ __forceinline__ float fast_exp2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ bool wait_raw(uint32_t bar, uint32_t parity, uint64_t budget_ns)
{
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity))
        if (globaltimer_ns() - t0 > budget_ns) return false;
    return true;
}

// 32 lanes x 32 bits, 32 consecutive columns: thread i gets lane (base + i).
__device__ __forceinline__ void tmem_ld_32x32b_x32(uint32_t taddr, uint32_t (&r)[32])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_st_32x32b_x32(uint32_t taddr, const uint32_t (&r)[32])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]),
        "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]),
        "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}

// Units of stream v (V streams): v, v + V, v + 2V, ...
__device__ __forceinline__ int stream_units(const DenseParams& p, int v, int V)
{
    return p.units > v ? (p.units - v + V - 1) / V : 0;
}

__global__ void __launch_bounds__(kThreads, 1) ssba_dense_tc_kernel(const __grid_constant__ DenseMaps maps,
                                                                    const __grid_constant__ DenseParams p)
{
    extern __shared__ uint8_t smem_raw[];
    DenseSmem& cs = *reinterpret_cast<DenseSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                  ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        cs.abort_flag = 0;
        for (int s = 0; s < kStreams; ++s) {
            StreamSmem& sm = cs.st[s];
            for (int b = 0; b < 2; ++b) {
                mbar_init(smem_u32(&sm.q_full[b]), 1);
                mbar_init(smem_u32(&sm.q_empty[b]), 1);
                mbar_init(smem_u32(&sm.stats_full[b]), 4);
                mbar_init(smem_u32(&sm.stats_free[b]), 4);
            }
            for (int b = 0; b < kStages; ++b) {
                mbar_init(smem_u32(&sm.k_full[b]), 1);
                mbar_init(smem_u32(&sm.k_empty[b]), 1);
                mbar_init(smem_u32(&sm.v_full[b]), 1);
                mbar_init(smem_u32(&sm.v_empty[b]), 1);
            }
            mbar_init(smem_u32(&sm.s_full), 1);
            mbar_init(smem_u32(&sm.s_free), 4);
            mbar_init(smem_u32(&sm.p_full), 4);
            mbar_init(smem_u32(&sm.p_empty), 1);
            mbar_init(smem_u32(&sm.o_full), 1);
            mbar_init(smem_u32(&sm.o_free), 4);
            mbar_init(smem_u32(&sm.drain[0]), 1);
            mbar_init(smem_u32(&sm.drain[1]), 1);
        }
        fence_mbar_init();
    }
    if (warp == 2) {
        tmem_alloc(smem_u32(&cs.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    if (warp < 2 && lane == 0) {
        tma_prefetch_desc(&maps.q);
        tma_prefetch_desc(&maps.k);
        tma_prefetch_desc(&maps.v);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // everything above reads no input (programmatic dependent launch: inputs may come from the
    // grid launched before this one)
    grid_dep_wait();
    grid_dep_launch();
    // roles: stream of the warp, and its role
    int stream, role;  // role 0 producer, 1 MMA, 2 softmax, 3 epilogue
    if (warp < 2) { stream = warp; role = 0; }
    else if (warp < 4) { stream = warp - 2; role = 1; }
    else if (warp < 12) { stream = (warp - 4) / 4; role = 2; }
    else { stream = (warp - 12) / 4; role = 3; }
    StreamSmem& sm = cs.st[stream];
    const int V = gridDim.x * kStreams;
    const int v = stream * gridDim.x + blockIdx.x;  // stream-major numbering of the grid's streams
    const int nunits = stream_units(p, v, V);
    const uint32_t tbase = cs.tmem_base + stream * kStreamCols;
    volatile int* abortf = &cs.abort_flag;
    bool dead = false;

    if (role == 0) {
        // ------------------------------------------------------------ TMA producer
        uint32_t gk = 0;  // key tiles loaded by this stream
        if (lane == 0) {
            for (int n = 0; n < nunits && !dead; ++n) {
                const int u = v + n * V, bh = u / p.nt, qt = u - bh * p.nt;
                const uint32_t qb = n & 1;
                if (!mbar_wait(smem_u32(&sm.q_empty[qb]), ((n >> 1) & 1) ^ 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                mbar_arrive_expect_tx(smem_u32(&sm.q_full[qb]), kTileBytes);
                tma_load_3d(smem_u32(&sm.q[qb][0]), &maps.q, smem_u32(&sm.q_full[qb]), 0, qt * kTile, bh);
                for (int j = 0; j < p.nt; ++j, ++gk) {
                    const uint32_t slot = gk % kStages, ph = ((gk / kStages) & 1) ^ 1;
                    if (!mbar_wait(smem_u32(&sm.k_empty[slot]), ph, abortf, p.budget_ns)) {
                        dead = true;
                        break;
                    }
                    mbar_arrive_expect_tx(smem_u32(&sm.k_full[slot]), kTileBytes);
                    tma_load_3d(smem_u32(&sm.k[slot][0]), &maps.k, smem_u32(&sm.k_full[slot]), 0, j * kTile, bh);
                    if (!mbar_wait(smem_u32(&sm.v_empty[slot]), ph, abortf, p.budget_ns)) {
                        dead = true;
                        break;
                    }
                    mbar_arrive_expect_tx(smem_u32(&sm.v_full[slot]), kTileBytes);
                    tma_load_3d(smem_u32(&sm.v[slot][0]), &maps.v, smem_u32(&sm.v_full[slot]), 0, j * kTile, bh);
                }
            }
            if (dead) {  // drain the copies that may still be in flight
                for (uint32_t x = gk > kStages ? gk - kStages : 0; x < gk; ++x) {
                    wait_raw(smem_u32(&sm.k_full[x % kStages]), (x / kStages) & 1, p.budget_ns);
                    wait_raw(smem_u32(&sm.v_full[x % kStages]), (x / kStages) & 1, p.budget_ns);
                }
            }
        }
        __syncwarp();
    } else if (role == 1) {
        // ------------------------------------------------------------ MMA issuer
        // QK_j into S once the softmax has loaded S_{j-1}; then PV_{j-1} once P_{j-1} is stored.
        const bool leader = elect_one_sync();
        uint32_t gs = 0, gp = 0;  // key tiles through S; through P
        auto do_pv = [&](int n, int j) -> bool {
            const uint32_t slot = gp % kStages;
            if (!mbar_wait(smem_u32(&sm.p_full), gp & 1, abortf, p.budget_ns)) return false;
            if (j == 0 && n > 0 && !mbar_wait(smem_u32(&sm.o_free), (n - 1) & 1, abortf, p.budget_ns)) return false;
            if (!mbar_wait(smem_u32(&sm.v_full[slot]), (gp / kStages) & 1, abortf, p.budget_ns)) return false;
            tc_fence_after();
            if (elect_one_sync()) {
                const uint64_t vdesc = sdesc_sw128(smem_u32(&sm.v[slot][0]), 8192, 1024);
#pragma unroll
                for (int k = 0; k < kTile / 16; ++k)
                    mma_ts(tbase + kColO, tbase + kColP + k * 8, vdesc + (uint64_t)(k * 128), kIdescPV,
                           (j > 0 || k > 0) ? 1u : 0u);
                mma_commit(smem_u32(&sm.v_empty[slot]));
                mma_commit(smem_u32(&sm.p_empty));
                if (j == p.nt - 1) mma_commit(smem_u32(&sm.o_full));
            }
            __syncwarp();
            ++gp;
            return true;
        };
        for (int n = 0; n < nunits && !dead; ++n) {
            const uint32_t qb = n & 1;
            if (!mbar_wait(smem_u32(&sm.q_full[qb]), (n >> 1) & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            for (int j = 0; j < p.nt; ++j, ++gs) {
                const uint32_t slot = gs % kStages;
                if (gs >= 1u && !mbar_wait(smem_u32(&sm.s_free), (gs - 1) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                if (!mbar_wait(smem_u32(&sm.k_full[slot]), (gs / kStages) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                if (elect_one_sync()) {
                    const uint64_t adesc = sdesc_sw128(smem_u32(&sm.q[qb][0]), 16, 1024);
                    const uint64_t bdesc = sdesc_sw128(smem_u32(&sm.k[slot][0]), 16, 1024);
#pragma unroll
                    for (int k = 0; k < kD / 16; ++k)
                        mma_ss(tbase + kColS, adesc + (uint64_t)(k * 2), bdesc + (uint64_t)(k * 2), kIdescQK,
                               k > 0 ? 1u : 0u);
                    mma_commit(smem_u32(&sm.s_full));
                    mma_commit(smem_u32(&sm.k_empty[slot]));
                    if (j == p.nt - 1) mma_commit(smem_u32(&sm.q_empty[qb]));
                }
                __syncwarp();
                if (j > 0 && !do_pv(n, j - 1)) {
                    dead = true;
                    break;
                }
            }
            if (dead) break;
            if (!do_pv(n, p.nt - 1)) {
                dead = true;
                break;
            }
        }
        if (dead && leader) {
            mma_commit(smem_u32(&sm.drain[0]));
            wait_raw(smem_u32(&sm.drain[0]), 0, p.budget_ns);
        }
    } else if (role == 2) {
        // ------------------------------------------------------------ softmax
        // Thread = row 32 quad + lane. Pass 1 reads the tile's 128 scores for the row maximum;
        // pass 2 reads them again for exp2(s c - m), the row sum and the bf16 P store.
        const int quad = warp & 3;
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        const uint32_t scol = tbase + lane_off + kColS, pcol = tbase + lane_off + kColP, ocol = tbase + lane_off + kColO;
        const float c = p.scale_log2;
        uint32_t gs = 0;
        for (int n = 0; n < nunits && !dead; ++n) {
            float m_used = 0.f, l = 0.f;
            for (int j = 0; j < p.nt; ++j, ++gs) {
                if (!mbar_wait(smem_u32(&sm.s_full), gs & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                float mx = -INFINITY;
#pragma unroll
                for (int ch = 0; ch < 4; ++ch) {
                    uint32_t a[32];
                    tmem_ld_32x32b_x32(scol + 32 * ch, a);
                    tmem_wait_ld();
                    float t4[4] = {mx, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                    for (int e = 0; e < 32; ++e) t4[e & 3] = fmaxf(t4[e & 3], __uint_as_float(a[e]));
                    mx = fmaxf(fmaxf(t4[0], t4[1]), fmaxf(t4[2], t4[3]));
                }
                const float mx2 = mx * c;
                // lazy rescale: the running max is raised only when it grows by more than
                // 2^kRescaleLog2 (warp-uniform decision: O is rescaled by a warp-wide TMEM access)
                bool rescale = false;
                float alpha = 1.f;
                if (j == 0) {
                    m_used = mx2;
                } else {
                    const bool need = mx2 > m_used + kRescaleLog2;
                    rescale = __any_sync(0xffffffffu, need);
                    if (need) {
                        alpha = fast_exp2(m_used - mx2);
                        m_used = mx2;
                    }
                }
                // the P buffer is free once PV_{j-1} has finished (O then holds every earlier PV)
                if (gs >= 1u && !mbar_wait(smem_u32(&sm.p_empty), (gs - 1) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                const float2 c2 = make_float2(c, c), nm2 = make_float2(-m_used, -m_used);
                float2 ls2 = make_float2(0.f, 0.f);
#pragma unroll
                for (int ch = 0; ch < 4; ++ch) {
                    uint32_t r[32];
                    tmem_ld_32x32b_x32(scol + 32 * ch, r);
                    tmem_wait_ld();
                    if (ch == 3) {  // S read in full: QK_{j+1} may overwrite it
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(smem_u32(&sm.s_free));
                    }
                    uint32_t pk[16];
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const float2 x = __ffma2_rn(make_float2(__uint_as_float(r[2 * e]), __uint_as_float(r[2 * e + 1])),
                                                    c2, nm2);
                        const float2 pp = make_float2(fast_exp2(x.x), fast_exp2(x.y));
                        ls2 = __fadd2_rn(ls2, pp);
                        pk[e] = pack_bf16(pp.x, pp.y);
                    }
                    tmem_st_32x32b_x16(pcol + 16 * ch, pk);
                }
                l = fmaf(l, alpha, ls2.x + ls2.y);
                if (rescale) {
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        uint32_t o[32];
                        tmem_ld_32x32b_x32(ocol + 32 * h, o);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                        tmem_st_32x32b_x32(ocol + 32 * h, o);
                    }
                }
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&sm.p_full));
            }
            if (dead) break;
            const uint32_t eb = n & 1;
            if (!mbar_wait(smem_u32(&sm.stats_free[eb]), ((n >> 1) & 1) ^ 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            sm.stats[eb][quad * 32 + lane] = make_float2(m_used, l);
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&sm.stats_full[eb]));
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int quad = warp & 3;
        const int row = quad * 32 + lane;
        const uint32_t ocol = tbase + (static_cast<uint32_t>(quad * 32) << 16) + kColO;
        for (int n = 0; n < nunits && !dead; ++n) {
            const int u = v + n * V, bh = u / p.nt, qt = u - bh * p.nt;
            if (!mbar_wait(smem_u32(&sm.o_full), n & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            // the row statistics first (the softmax hands them over after its last tile, before
            // the last PV has finished), then O in two halves of 32 columns
            const uint32_t eb = n & 1;
            if (!mbar_wait(smem_u32(&sm.stats_full[eb]), (n >> 1) & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            const float2 st = sm.stats[eb][row];
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&sm.stats_free[eb]));
            const bool ok = st.y > 0.f;
            const float inv = ok ? 1.f / st.y : 0.f;
            const size_t tok = (size_t)bh * p.N + (size_t)qt * kTile + row;
            uint4* dst = reinterpret_cast<uint4*>(p.O + tok * kD);
            tc_fence_after();
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                uint32_t o[32];
                tmem_ld_32x32b_x32(ocol + 32 * h, o);
                tmem_wait_ld();
                if (h == 1) {  // O read in full: the next unit's first PV may overwrite it
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(smem_u32(&sm.o_free));
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    uint4 w;
                    w.x = pack_bf16(__uint_as_float(o[8 * i + 0]) * inv, __uint_as_float(o[8 * i + 1]) * inv);
                    w.y = pack_bf16(__uint_as_float(o[8 * i + 2]) * inv, __uint_as_float(o[8 * i + 3]) * inv);
                    w.z = pack_bf16(__uint_as_float(o[8 * i + 4]) * inv, __uint_as_float(o[8 * i + 5]) * inv);
                    w.w = pack_bf16(__uint_as_float(o[8 * i + 6]) * inv, __uint_as_float(o[8 * i + 7]) * inv);
                    dst[4 * h + i] = w;
                }
            }
            p.lse[tok] = ok ? (st.x * 0.69314718055994531f + logf(st.y)) : -INFINITY;
        }
    }
    if (dead) atomicExch(p.status, SSBA_ERR_TIMEOUT);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 2) tmem_dealloc(cs.tmem_base, kTmemCols);
}

// [B*heads][N][64] bf16 as a 3-D map with 128-row boxes (128-byte swizzle).
bool encode_tile_map(CUtensorMap* m, const void* base, int BH, int N)
{
    EncodeTiledFn fn = tensor_map_encoder();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)N, (cuuint64_t)BH};
    cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)N * kD * 2};
    cuuint32_t box[3] = {kD, kTile, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

PerDeviceOnce g_dense_attr;

}  // namespace

int launch_dense_m128(const ssba_desc& d, float scale, const void* Q, const void* K, const void* V, void* O,
                      float* lse, cudaStream_t st)
{
    const long long N = (long long)d.H_tok * d.W_tok;
    const int BH = d.B * d.heads;
    if (d.head_dim != kD || d.dtype != SSBA_BF16 || N % kTile != 0 || N >= (1LL << 30)) return SSBA_ERR_UNSUPPORTED;
    DenseMaps maps;
    memset(&maps, 0, sizeof(maps));
    if (!encode_tile_map(&maps.q, Q, BH, (int)N) || !encode_tile_map(&maps.k, K, BH, (int)N) ||
        !encode_tile_map(&maps.v, V, BH, (int)N)) {
        set_error("ssba_forward_dense: cuTensorMapEncodeTiled failed");
        return SSBA_ERR_CUDA;
    }
    DenseParams p;
    p.O = static_cast<__nv_bfloat16*>(O);
    p.lse = lse;
    p.BH = BH;
    p.N = (int)N;
    p.nt = (int)(N / kTile);
    p.units = BH * p.nt;
    p.scale_log2 = scale * 1.4426950408889634f;
    p.status = device_status_word();
    p.budget_ns = kWaitBudgetNs;
    if (!p.status) {
        set_error("ssba_forward_dense: could not resolve the device status word");
        return SSBA_ERR_CUDA;
    }
    const size_t smem = sizeof(DenseSmem) + 1024;
    g_dense_attr.run([smem] {
        cudaFuncSetAttribute(ssba_dense_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    });
    const int want = (p.units + kStreams - 1) / kStreams;
    const int sms = device_sm_count();
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(want < sms ? want : sms, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, ssba_dense_tc_kernel, maps, p);
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("ssba_dense_tc_kernel launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

}  // namespace ssba
