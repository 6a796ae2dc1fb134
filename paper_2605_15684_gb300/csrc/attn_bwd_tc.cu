// attn_bwd_tc.cu -- gradients of the block-sparse attention (the backward of Algorithm 1's
// SparseAttention over the same kept blocks) on the sm_103a tensor cores, bf16 inputs.
//
// For the output gradient dO, with p_nm = exp(scale q_n.k_m - lse_n) over the kept pairs:
//   D_n = dO_n . O_n,  ds_nm = p_nm (dO_n . v_m - D_n),
//   dQ_n = scale sum_m ds_nm k_m,  dK_m = scale sum_n ds_nm q_n,  dV_m = sum_n p_nm dO_n.
// Deterministic (no atomics). A row kernel writes D for every row; then one grid holds both
// gradient roles, one (batch*head, block) per CTA, launched as a programmatic dependent of the
// row kernel (only the key-block role waits for D). Each 64 x 64 tile product is a
// tcgen05.mma kind::f16 with M=64 (four K=16 steps).
// 160 threads: warps 0-3 own the TMEM lane quadrants (the exps, the bf16 operands, the tile
// copies, the epilogue); lane 0 of warp 4 issues every MMA, so that issuing (some 80 cycles
// an instruction) runs beside the compute warps instead of in front of them. The two sides
// meet on mbarriers: MMA commits one way, one arrive per compute warp the other.
//   dq_block     query block i: for each kept key block j (list order)
//                              S  = Q_i K_j^T,  dP = dO_i V_j^T        (A, B from shared memory)
//                              dS = P o (dP - D) in registers, bf16 into shared memory
//                              dQ += dS K_j                           (B read MN-major)
//   dkdv_block   key block j: for each query block i whose list holds j (ascending)
//                              S^T = K_j Q_i^T,  dP^T = V_j dO_i^T
//                              P^T, dS^T in registers, bf16 into shared memory
//                              dV += P^T dO_i,  dK += dS^T Q_i
// Tiles are gathered token by token (the shifted window) with 16-byte cp.async into the
// 128-byte-swizzled layout the MMA descriptors read (K-major for A/B, MN-major as the second
// operand of the accumulating products), in three buffers: pair t computes, pair t + 1's tiles
// are resident and pair t + 2's are in flight. S_{t+1} and dP_{t+1} are issued as soon as
// S_t and dP_t are in registers, so the tensor core runs the next pair's products while the
// threads form this pair's bf16 operands. TMEM: S, dP and one or two fp32 accumulators
// (256 columns, two CTAs per SM). The thread that owns TMEM lane (row) r of the M=64 data
// path holds half a row: columns [32 h, 32 h + 32), h = lane / 16. Every mbarrier wait is
// bounded; a timeout is written to the device status word and the CTA drains its MMAs before
// it exits.
#include <cstdint>

#include "common.cuh"
#include "bwd_tile.cuh"
#include "ptx.cuh"
#include "window.cuh"

namespace ssba {

namespace {

using namespace ptx;

using namespace bwd;

constexpr int kCompute = 128;  // warps 0-3: one TMEM lane quadrant each
constexpr int kThreads = 160;  // + warp 4, whose lane 0 issues every MMA of the CTA
constexpr int kIssuer = 128;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColS = 0, kColDP = 64, kColA0 = 128, kColA1 = 192;
constexpr size_t kSmemBytes = 100 * 1024;  // also keeps residency at two CTAs per SM (TMEM)

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Token of in-window position pos of the window whose unshifted origin is (r0, c0) (the map of
// Grid::token with blk = 8, the window origin computed once per tile).
struct WinOrigin {
    int r0, c0;
};
__device__ __forceinline__ WinOrigin win_origin(const Grid& g, int label)
{
    const int br = label / g.bw, bc = label - br * g.bw;
    int r0 = br * 8 - g.sr, c0 = bc * 8 - g.sc;
    r0 += r0 < 0 ? g.H : 0;
    c0 += c0 < 0 ? g.W : 0;
    return {r0, c0};
}
__device__ __forceinline__ int win_token(const Grid& g, WinOrigin o, int pos)
{
    int r = o.r0 + (pos >> 3), c = o.c0 + (pos & 7);
    r -= r >= g.H ? g.H : 0;
    c -= c >= g.W ? g.W : 0;
    return r * g.W + c;
}

// Block `label` of a [N][64] bf16 head into a 1024-aligned 8 KB tile: row r = in-window
// position r, 16-byte chunk c at chunk c ^ (r & 7) (the 128-byte swizzle). Called by the
// compute threads.
__device__ __forceinline__ void load_tile(uint32_t dst, const __nv_bfloat16* X, const Grid& g, int label)
{
    const WinOrigin o = win_origin(g, label);
#pragma unroll
    for (int i = 0; i < kT * 8 / kCompute; ++i) {
        const int e = threadIdx.x + i * kCompute, r = e >> 3, c = e & 7;
        cp_async16(dst + r * 128 + ((c ^ (r & 7)) << 4), X + (size_t)win_token(g, o, r) * kD + c * 8);
    }
}

struct alignas(1024) BwdSmem {
    uint8_t a[kTile];        // dq: Q_i;  dkdv: K_j
    uint8_t b[kTile];        // dq: dO_i; dkdv: V_j
    uint8_t x[3][kTile];     // dq: K_j;  dkdv: Q_i   (three buffers: pair t computes, t + 1 is
    uint8_t y[3][kTile];     // dq: V_j;  dkdv: dO_i   loaded, t + 2 is being copied)
    uint8_t e[2][kTile];     // dq: dS (e[0]); dkdv: P^T, dS^T -- bf16, the A operands of the
                             // accumulating products, written from registers
    float ls[3][kT];         // dkdv: lse of the query block
    float ds[3][kT];         // dkdv: D of the query block
    int list[256];           // dkdv: the query blocks holding this key block, ascending
    int wcount[kThreads / 32];
    uint64_t bar_s, bar_a, drain;  // MMA commits: S and dP ready; accumulators updated; drain
    uint64_t full_s, full_a;       // compute warps (one arrive each): S, dP read and the next
                                   // tiles landed; the bf16 operands stored
    uint32_t tmem_base;
    int abort_flag;
};
static_assert(sizeof(BwdSmem) + 1024 <= kSmemBytes, "shared memory");

__device__ __forceinline__ BwdSmem& smem_layout()
{
    extern __shared__ uint8_t raw[];
    return *reinterpret_cast<BwdSmem*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~static_cast<uintptr_t>(1023));
}

__device__ __forceinline__ void setup(BwdSmem& sm)
{
    if (threadIdx.x == 0) {
        sm.abort_flag = 0;
        mbar_init(smem_u32(&sm.bar_s), 1);
        mbar_init(smem_u32(&sm.bar_a), 1);
        mbar_init(smem_u32(&sm.drain), 1);
        mbar_init(smem_u32(&sm.full_s), kCompute / 32);
        mbar_init(smem_u32(&sm.full_a), kCompute / 32);
        fence_mbar_init();
    }
    if (threadIdx.x < 32) {
        tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
}

__device__ __forceinline__ void teardown(BwdSmem& sm, const BwdParams& p, bool dead, uint32_t issued)
{
    cp_async_wait<0>();
    if (dead) {
        if (threadIdx.x == kIssuer && issued) {  // the MMAs still in flight
            mma_commit(smem_u32(&sm.drain));
            const uint64_t t0 = globaltimer_ns();
            while (!mbar_try_wait(smem_u32(&sm.drain), 0) && globaltimer_ns() - t0 < p.budget_ns) {
            }
        }
        if (threadIdx.x == 0) atomicExch(p.status, SSBA_ERR_TIMEOUT);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (threadIdx.x < 32) tmem_dealloc(sm.tmem_base, kTmemCols);
}

// A compute warp's bounded wait: the warp goes on only if every lane saw the phase, so that a
// timeout takes the whole warp out of the loop at once.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abortf, uint64_t budget_ns)
{
    const bool ok = mbar_wait(bar, parity, abortf, budget_ns);
    return __all_sync(0xffffffffu, ok);
}

// One arrive per compute warp, after every lane's TMEM loads and shared-memory writes.
__device__ __forceinline__ void warp_arrive(uint32_t bar)
{
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}

// Writes the 64 x 64 fp32 accumulator at TMEM column `col`, times `mul`, to rows
// g.token(label, r) of out (one [N][64] head).
__device__ __forceinline__ void store_acc(uint32_t taddr, float* out, const Grid& g, int label, float mul)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, h = lane >> 4;
    const int r = warp * 16 + (lane & 15);
    uint32_t v[32];
    tmem_ld_16x32bx2_x16_off32(taddr, *reinterpret_cast<uint32_t(*)[16]>(&v[0]));
    tmem_ld_16x32bx2_x16_off32(taddr + 16, *reinterpret_cast<uint32_t(*)[16]>(&v[16]));
    tmem_wait_ld();
    float4* dst = reinterpret_cast<float4*>(out + (size_t)g.token(label, r) * kD + 32 * h);
#pragma unroll
    for (int i = 0; i < 8; ++i)
        dst[i] = make_float4(__uint_as_float(v[4 * i]) * mul, __uint_as_float(v[4 * i + 1]) * mul,
                             __uint_as_float(v[4 * i + 2]) * mul, __uint_as_float(v[4 * i + 3]) * mul);
}

// dQ of query block `label` of head bh (D comes from the row kernel; computed here again
// for this block's own rows, so that this role needs nothing from that kernel).
__device__ __forceinline__ void dq_block(const BwdParams& p, const int label, const int bh)
{
    BwdSmem& sm = smem_layout();
    const Grid g = p.g;
    const int Tb = g.Tb(), N = g.H * g.W;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, h = lane >> 4;
    const int r = (warp & 3) * 16 + (lane & 15);  // tile row of a compute thread
    const size_t head = (size_t)bh * N * kD;
    const size_t row = (size_t)bh * N + g.token(label, r);
    volatile int* abortf = &sm.abort_flag;
    // the kept key blocks into shared memory (visible after the set-up's barrier)
    const int32_t* list = p.idx + ((size_t)bh * Tb + label) * p.keep;
    const int n = min(max(p.cnt[(size_t)bh * Tb + label], 0), p.keep);
    for (int i = threadIdx.x; i < n; i += kThreads) sm.list[i] = min(max(__ldg(list + i), 0), Tb - 1);
    setup(sm);
    const uint32_t tb = sm.tmem_base + (static_cast<uint32_t>((warp & 3) * 32) << 16);
    const uint32_t tb0 = sm.tmem_base;
    bool dead = false;
    uint32_t issued = 0;

    if (threadIdx.x < kCompute) {
        // tiles of pair t in buffer t % 3: K_j in x, V_j in y
        auto fetch = [&](int t) {
            const int j = sm.list[t];
            load_tile(smem_u32(sm.x[t % 3]), p.K + head, g, j);
            load_tile(smem_u32(sm.y[t % 3]), p.V + head, g, j);
            cp_async_commit();
        };
        load_tile(smem_u32(sm.a), p.Q + head, g, label);
        load_tile(smem_u32(sm.b), p.dO + head, g, label);
        cp_async_commit();
        if (n > 0) fetch(0);
        if (n > 1) fetch(1);

        // D for this row (both halves of the row's threads hold it) and the log2-domain lse,
        // while the tiles are in flight
        float Dr = 0.f;
        {
            const uint4* go = reinterpret_cast<const uint4*>(p.dO + row * kD + 32 * h);
            const uint4* oo = reinterpret_cast<const uint4*>(p.O + row * kD + 32 * h);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint4 a = __ldg(go + i), b = __ldg(oo + i);
                const uint32_t aw[4] = {a.x, a.y, a.z, a.w}, bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float2 fa = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&aw[k]));
                    const float2 fb = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bw[k]));
                    Dr = fmaf(fa.x, fb.x, Dr);
                    Dr = fmaf(fa.y, fb.y, Dr);
                }
            }
        }
        Dr += __shfl_xor_sync(0xffffffffu, Dr, 16);
        const float c = p.scale * kLog2e;
        const float L2 = p.lse[row] * kLog2e;
        if (n > 0) {  // Q, dO and the tiles of pair 0 landed
            if (n > 1) cp_async_wait<1>(); else cp_async_wait<0>();
            fence_proxy_async_smem();
            warp_arrive(smem_u32(&sm.full_s));
        }
        // Pair t: S_t, dP_t into registers, then the issuer may overwrite them with pair t + 1's
        // products; dS_t goes to shared memory once dQ_{t-1} has read the last one.
        for (int t = 0; t < n; ++t) {
            if (!warp_wait(smem_u32(&sm.bar_s), t & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            tc_fence_after();
            uint32_t s[32], dp[32];
            tmem_ld_16x32bx2_x16_off32(tb + kColS, *reinterpret_cast<uint32_t(*)[16]>(&s[0]));
            tmem_ld_16x32bx2_x16_off32(tb + kColS + 16, *reinterpret_cast<uint32_t(*)[16]>(&s[16]));
            tmem_ld_16x32bx2_x16_off32(tb + kColDP, *reinterpret_cast<uint32_t(*)[16]>(&dp[0]));
            tmem_ld_16x32bx2_x16_off32(tb + kColDP + 16, *reinterpret_cast<uint32_t(*)[16]>(&dp[16]));
            tmem_wait_ld();
            tc_fence_before();
            if (t + 1 < n) {  // the tiles of pair t + 1 (copied during pair t - 1)
                cp_async_wait<0>();
                fence_proxy_async_smem();
            }
            warp_arrive(smem_u32(&sm.full_s));
            uint32_t pk[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const float p0 = fast_exp2(fmaf(__uint_as_float(s[2 * i]), c, -L2));
                const float p1 = fast_exp2(fmaf(__uint_as_float(s[2 * i + 1]), c, -L2));
                pk[i] = pack_bf16(p0 * (__uint_as_float(dp[2 * i]) - Dr), p1 * (__uint_as_float(dp[2 * i + 1]) - Dr));
            }
            // dQ_{t-1} has read the last dS and the tiles of pair t - 1
            if (t >= 1 && !warp_wait(smem_u32(&sm.bar_a), (t - 1) & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            if (t + 2 < n) fetch(t + 2);  // into the buffers of pair t - 1
            store_half_row(sm.e[0], r, h, pk);
            fence_proxy_async_smem();
            warp_arrive(smem_u32(&sm.full_a));
        }
        if (!dead && n > 0 && !warp_wait(smem_u32(&sm.bar_a), (n - 1) & 1, abortf, p.budget_ns)) dead = true;
    } else if (threadIdx.x == kIssuer && n > 0) {
        // S_0, dP_0; then per pair t: S_{t+1}, dP_{t+1} once S_t, dP_t are in registers, and
        // dQ += dS_t K_t once dS_t is stored
        if (mbar_wait(smem_u32(&sm.full_s), 0, abortf, p.budget_ns)) {
            tc_fence_after();
            mma_kk(tb0 + kColS, smem_u32(sm.a), smem_u32(sm.x[0]));   // S = Q K^T
            mma_kk(tb0 + kColDP, smem_u32(sm.b), smem_u32(sm.y[0]));  // dP = dO V^T
            mma_commit(smem_u32(&sm.bar_s));
            issued = 1;
            for (int t = 0; t < n; ++t) {
                if (!mbar_wait(smem_u32(&sm.full_s), (t + 1) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                if (t + 1 < n) {
                    mma_kk(tb0 + kColS, smem_u32(sm.a), smem_u32(sm.x[(t + 1) % 3]));
                    mma_kk(tb0 + kColDP, smem_u32(sm.b), smem_u32(sm.y[(t + 1) % 3]));
                    mma_commit(smem_u32(&sm.bar_s));
                }
                if (!mbar_wait(smem_u32(&sm.full_a), t & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                mma_sb(tb0 + kColA0, smem_u32(sm.e[0]), smem_u32(sm.x[t % 3]), t > 0);  // dQ += dS K
                mma_commit(smem_u32(&sm.bar_a));
            }
        } else {
            dead = true;
        }
    }
    dead = __syncthreads_or(dead);
    if (!dead && threadIdx.x < kCompute) {
        tc_fence_after();
        if (n > 0) {
            store_acc(tb + kColA0, p.dQ + head, g, label, p.scale);
        } else {
            float4* dst = reinterpret_cast<float4*>(p.dQ + row * kD + 32 * h);
#pragma unroll
            for (int i = 0; i < 8; ++i) dst[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    teardown(sm, p, dead, issued);
}

// dK, dV of key block `label` of head bh.
__device__ __forceinline__ void dkdv_block(const BwdParams& p, const int label, const int bh)
{
    BwdSmem& sm = smem_layout();
    const Grid g = p.g;
    const int Tb = g.Tb(), N = g.H * g.W;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, h = lane >> 4;
    const int r = (warp & 3) * 16 + (lane & 15);  // tile row of a compute thread
    const size_t head = (size_t)bh * N * kD;
    volatile int* abortf = &sm.abort_flag;
    const float c = p.scale * kLog2e;

    if (threadIdx.x < kCompute) {
        load_tile(smem_u32(sm.a), p.K + head, g, label);
        load_tile(smem_u32(sm.b), p.V + head, g, label);
        cp_async_commit();
    }

    // the query blocks whose lists hold this key block, ascending
    int total = 0;
    for (int i0 = 0; i0 < Tb; i0 += kThreads) {
        const int i = i0 + threadIdx.x;
        bool has = false;
        if (i < Tb) {
            const int32_t* l = p.idx + ((size_t)bh * Tb + i) * p.keep;
            const int nn = min(max(p.cnt[(size_t)bh * Tb + i], 0), p.keep);
            // four list entries in flight at a time
            for (int t = 0; t < nn; t += 4) {
                int v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) v[u] = t + u < nn ? __ldg(l + t + u) : -1;
#pragma unroll
                for (int u = 0; u < 4; ++u) has |= v[u] == label;
            }
        }
        const unsigned b = __ballot_sync(0xffffffffu, has);
        __syncthreads();
        if (lane == 0) sm.wcount[warp] = __popc(b);
        __syncthreads();
        int off = total;
        for (int w = 0; w < warp; ++w) off += sm.wcount[w];
        if (has) sm.list[off + __popc(b & ((1u << lane) - 1u))] = i;
        for (int w = 0; w < kThreads / 32; ++w) total += sm.wcount[w];
    }
    const int n = total;
    setup(sm);  // its barrier also publishes the list
    const uint32_t tb = sm.tmem_base + (static_cast<uint32_t>((warp & 3) * 32) << 16);
    const uint32_t tb0 = sm.tmem_base;
    bool dead = false;
    uint32_t issued = 0;

    if (threadIdx.x < kCompute) {
        // tiles of pair t in buffer t % 3: Q_i in x, dO_i in y, and the block's lse and D
        auto fetch = [&](int t) {
            const int qi = sm.list[t], buf = t % 3;
            load_tile(smem_u32(sm.x[buf]), p.Q + head, g, qi);
            load_tile(smem_u32(sm.y[buf]), p.dO + head, g, qi);
            if (threadIdx.x < kT) {
                const size_t qrow = (size_t)bh * N + win_token(g, win_origin(g, qi), threadIdx.x);
                cp_async4(smem_u32(&sm.ls[buf][threadIdx.x]), p.lse + qrow);
                cp_async4(smem_u32(&sm.ds[buf][threadIdx.x]), p.Dbuf + qrow);
            }
            cp_async_commit();
        };
        grid_dep_wait();  // D of every row, from the row kernel
        if (n > 0) fetch(0);
        if (n > 1) fetch(1);
        if (n > 0) {  // K, V and the tiles of pair 0 landed
            if (n > 1) cp_async_wait<1>(); else cp_async_wait<0>();
            fence_proxy_async_smem();
            warp_arrive(smem_u32(&sm.full_s));
        }
        // Pair t as in the dQ kernel, with P^T_t and dS^T_t as the stored operands.
        for (int t = 0; t < n; ++t) {
            const int buf = t % 3;
            if (!warp_wait(smem_u32(&sm.bar_s), t & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            tc_fence_after();
            uint32_t s[32], dp[32];
            tmem_ld_16x32bx2_x16_off32(tb + kColS, *reinterpret_cast<uint32_t(*)[16]>(&s[0]));
            tmem_ld_16x32bx2_x16_off32(tb + kColS + 16, *reinterpret_cast<uint32_t(*)[16]>(&s[16]));
            tmem_ld_16x32bx2_x16_off32(tb + kColDP, *reinterpret_cast<uint32_t(*)[16]>(&dp[0]));
            tmem_ld_16x32bx2_x16_off32(tb + kColDP + 16, *reinterpret_cast<uint32_t(*)[16]>(&dp[16]));
            tmem_wait_ld();
            tc_fence_before();
            if (t + 1 < n) {
                cp_async_wait<0>();
                fence_proxy_async_smem();
            }
            warp_arrive(smem_u32(&sm.full_s));
            // columns are the query rows 32 h + i of the block
            const float* Lq = sm.ls[buf] + 32 * h;
            const float* Dq = sm.ds[buf] + 32 * h;
            uint32_t pp[16], dd[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const float p0 = fast_exp2(fmaf(__uint_as_float(s[2 * i]), c, -Lq[2 * i] * kLog2e));
                const float p1 = fast_exp2(fmaf(__uint_as_float(s[2 * i + 1]), c, -Lq[2 * i + 1] * kLog2e));
                pp[i] = pack_bf16(p0, p1);
                dd[i] = pack_bf16(p0 * (__uint_as_float(dp[2 * i]) - Dq[2 * i]),
                                  p1 * (__uint_as_float(dp[2 * i + 1]) - Dq[2 * i + 1]));
            }
            if (t >= 1 && !warp_wait(smem_u32(&sm.bar_a), (t - 1) & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            if (t + 2 < n) fetch(t + 2);  // into the buffers of pair t - 1
            store_half_row(sm.e[0], r, h, pp);
            store_half_row(sm.e[1], r, h, dd);
            fence_proxy_async_smem();
            warp_arrive(smem_u32(&sm.full_a));
        }
        if (!dead && n > 0 && !warp_wait(smem_u32(&sm.bar_a), (n - 1) & 1, abortf, p.budget_ns)) dead = true;
    } else if (threadIdx.x == kIssuer && n > 0) {
        if (mbar_wait(smem_u32(&sm.full_s), 0, abortf, p.budget_ns)) {
            tc_fence_after();
            mma_kk(tb0 + kColS, smem_u32(sm.a), smem_u32(sm.x[0]));   // S^T = K Q^T
            mma_kk(tb0 + kColDP, smem_u32(sm.b), smem_u32(sm.y[0]));  // dP^T = V dO^T
            mma_commit(smem_u32(&sm.bar_s));
            issued = 1;
            for (int t = 0; t < n; ++t) {
                if (!mbar_wait(smem_u32(&sm.full_s), (t + 1) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                if (t + 1 < n) {
                    mma_kk(tb0 + kColS, smem_u32(sm.a), smem_u32(sm.x[(t + 1) % 3]));
                    mma_kk(tb0 + kColDP, smem_u32(sm.b), smem_u32(sm.y[(t + 1) % 3]));
                    mma_commit(smem_u32(&sm.bar_s));
                }
                if (!mbar_wait(smem_u32(&sm.full_a), t & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                mma_sb(tb0 + kColA0, smem_u32(sm.e[0]), smem_u32(sm.y[t % 3]), t > 0);  // dV += P^T dO
                mma_sb(tb0 + kColA1, smem_u32(sm.e[1]), smem_u32(sm.x[t % 3]), t > 0);  // dK += dS^T Q
                mma_commit(smem_u32(&sm.bar_a));
            }
        } else {
            dead = true;
        }
    }
    dead = __syncthreads_or(dead);
    if (!dead && threadIdx.x < kCompute) {
        tc_fence_after();
        if (n > 0) {
            store_acc(tb + kColA0, p.dV + head, g, label, 1.0f);
            store_acc(tb + kColA1, p.dK + head, g, label, p.scale);
        } else {
            const size_t krow = (size_t)bh * N + g.token(label, r);
            float4* a = reinterpret_cast<float4*>(p.dV + krow * kD + 32 * h);
            float4* b = reinterpret_cast<float4*>(p.dK + krow * kD + 32 * h);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                a[i] = make_float4(0.f, 0.f, 0.f, 0.f);
                b[i] = make_float4(0.f, 0.f, 0.f, 0.f);
            }
        }
    }
    teardown(sm, p, dead, issued);
}

// Head bh's transposed lists (see BwdParams): a bit per (key block j, query block i) in shared
// memory, then per key block its count, an exclusive scan over the key blocks, and its query
// blocks written in ascending order. Thread j owns key block j (Tb <= 256 = the block size).
__device__ __forceinline__ void build_transposed(const BwdParams& p, const int bh)
{
    __shared__ uint32_t bits[256 * 8];  // [j][i / 32]
    __shared__ int wsum[8];
    const int Tb = p.g.Tb(), nw = (Tb + 31) >> 5;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int w = threadIdx.x; w < Tb * nw; w += 256) bits[w] = 0;
    if (bh == 0 && threadIdx.x == 0) *p.ctr = 0;  // read by the gradient kernel after its wait
    __syncthreads();
    const int32_t* idx = p.idx + (size_t)bh * Tb * p.keep;
    const int32_t* cnt = p.cnt + (size_t)bh * Tb;
    for (int e = threadIdx.x; e < Tb * p.keep; e += 256) {
        const int i = e / p.keep, t = e - i * p.keep;
        if (t < min(max(__ldg(cnt + i), 0), p.keep)) {
            const int j = min(max(__ldg(idx + e), 0), Tb - 1);
            atomicOr(&bits[j * nw + (i >> 5)], 1u << (i & 31));
        }
    }
    __syncthreads();
    const int j = threadIdx.x;
    int c = 0;
    if (j < Tb)
        for (int w = 0; w < nw; ++w) c += __popc(bits[j * nw + w]);
    int v = c;  // inclusive scan within the warp, then over the warps
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += u;
    }
    if (lane == 31) wsum[warp] = v;
    __syncthreads();
    int off = v - c;
    for (int w = 0; w < warp; ++w) off += wsum[w];
    if (j < Tb) {
        const size_t row = (size_t)bh * Tb + j;
        p.toff[row] = (int)((size_t)bh * Tb * p.keep) + off;
        p.tcnt[row] = c;
        int* out = p.tlist + (size_t)bh * Tb * p.keep + off;
        for (int w = 0; w < nw; ++w) {
            uint32_t m = bits[j * nw + w];
            while (m) {
                const int b = __ffs(m) - 1;
                m &= m - 1;
                *out++ = w * 32 + b;
            }
        }
    }
}

// D_n = dO_n . O_n for every row, two threads a row (32 dims each); CTAs past row_blocks
// build the transposed lists, one head each.
__global__ void __launch_bounds__(256) ssba_bwd_rows_kernel(const BwdParams p, const int rows, const int row_blocks)
{
    grid_dep_launch();  // the gradient kernel's prologues need nothing from here
    if ((int)blockIdx.x >= row_blocks) {
        build_transposed(p, (int)blockIdx.x - row_blocks);
        return;
    }
    const int t = blockIdx.x * 256 + threadIdx.x;
    const int row = t >> 1, h = t & 1;
    float Dr = 0.f;
    if (row < rows) {
        const uint4* go = reinterpret_cast<const uint4*>(p.dO + (size_t)row * kD + 32 * h);
        const uint4* oo = reinterpret_cast<const uint4*>(p.O + (size_t)row * kD + 32 * h);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const uint4 a = __ldg(go + i), b = __ldg(oo + i);
            const uint32_t aw[4] = {a.x, a.y, a.z, a.w}, bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float2 fa = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&aw[k]));
                const float2 fb = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&bw[k]));
                Dr = fmaf(fa.x, fb.x, Dr);
                Dr = fmaf(fa.y, fb.y, Dr);
            }
        }
    }
    Dr += __shfl_xor_sync(0xffffffffu, Dr, 1);
    if (row < rows && h == 0) {
        p.Dbuf[row] = Dr;
        if (p.ld) {  // the same row by block, at its tile row, beside its log2-domain lse
            const int N = p.g.H * p.g.W, bh = row / N;
            int label, pos;
            win::token_block(p.g, row - bh * N, label, pos);
            const int r = win::tile_row_of(p.g, label, pos);
            p.ld[((size_t)bh * p.g.Tb() + label) * kT + r] = make_float2(__ldg(p.lse + row) * kLog2e, Dr);
        }
    }
}

// Both gradient roles in one grid: CTAs [0, BH Tb) are key blocks (dK, dV; their list lengths
// vary), the rest query blocks (dQ; all the same length), so that the query blocks fill in
// behind the key blocks instead of ending in a partial wave of their own.
__global__ void __launch_bounds__(kThreads) ssba_bwd_tc_kernel(const BwdParams p)
{
    const int Tb = p.g.Tb();
    const int nk = (int)(gridDim.x >> 1);
    const int item = blockIdx.x < nk ? blockIdx.x : blockIdx.x - nk;
    const int bh = item / Tb, label = item - bh * Tb;
    if ((int)blockIdx.x < nk)
        dkdv_block(p, label, bh);
    else
        dq_block(p, label, bh);
}

}  // namespace

namespace bwd {

BwdLayout bwd_layout(const ssba_desc& d, const Grid& g, int keep)
{
    auto up = [](size_t x) { return (x + 255) & ~static_cast<size_t>(255); };
    const size_t BH = (size_t)d.B * d.heads, Tb = (size_t)g.Tb();
    BwdLayout l;
    l.ctr = up(BH * g.H * g.W * sizeof(float));
    l.toff = l.ctr + 256;
    l.tcnt = l.toff + up(BH * Tb * sizeof(int));
    l.tlist = l.tcnt + up(BH * Tb * sizeof(int));
    l.ld = l.tlist + up(BH * Tb * (size_t)keep * sizeof(int));
    l.bytes = l.ld + up(BH * g.H * g.W * 2 * sizeof(float));
    return l;
}

cudaError_t launch_bwd_rows(const BwdParams& p, int BH, cudaStream_t st)
{
    const int rows = BH * p.g.H * p.g.W;
    const int row_blocks = (int)((2 * (size_t)rows + 255) / 256);
    const int extra = p.tlist ? BH : 0;
    ssba_bwd_rows_kernel<<<(unsigned)(row_blocks + extra), 256, 0, st>>>(p, rows, row_blocks);
    return cudaGetLastError();
}

}  // namespace bwd

int launch_backward_tc(const ssba_desc& d, const Grid& g, int keep, float scale, const void* Q, const void* K,
                       const void* V, const void* O, const float* lse, const void* dO, const int32_t* idx,
                       const int32_t* cnt, float* dQ, float* dK, float* dV, float* Dbuf, cudaStream_t st)
{
    if (d.head_dim != kD || g.blk != 8 || d.dtype != SSBA_BF16 || g.Tb() > 256) return SSBA_ERR_UNSUPPORTED;
    BwdParams p;
    p.Q = static_cast<const __nv_bfloat16*>(Q);
    p.K = static_cast<const __nv_bfloat16*>(K);
    p.V = static_cast<const __nv_bfloat16*>(V);
    p.O = static_cast<const __nv_bfloat16*>(O);
    p.dO = static_cast<const __nv_bfloat16*>(dO);
    p.lse = lse;
    p.idx = idx;
    p.cnt = cnt;
    p.dQ = dQ;
    p.dK = dK;
    p.dV = dV;
    p.Dbuf = Dbuf;
    p.ctr = p.toff = p.tcnt = p.tlist = nullptr;
    p.ld = nullptr;
    p.withhold = 0;
    p.g = g;
    p.keep = keep;
    p.scale = scale;
    p.budget_ns = kWaitBudgetNs;
    p.status = device_status_word();
    if (!p.status) {
        set_error("ssba_backward: could not resolve the device status word");
        return SSBA_ERR_CUDA;
    }
    static PerDeviceOnce attr;  // shared-memory attribute, set once per device
    attr.run([] {
        cudaFuncSetAttribute(ssba_bwd_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    });
    const int BH = d.B * d.heads;
    cudaError_t e = launch_bwd_rows(p, BH, st);
    if (e == cudaSuccess) {
        // launched as a programmatic dependent of the row kernel: only the key-block role waits
        // for it (grid_dep_wait before it reads D)
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)(2 * BH * g.Tb()));
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = kSmemBytes;
        cfg.stream = st;
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        at[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, ssba_bwd_tc_kernel, p);
    }
    if (e != cudaSuccess) {
        set_error("ssba_backward (tensor cores) launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

}  // namespace ssba
