// attn_bwd_ws.cu -- the tensor-core backward (gradients of Algorithm 1's SparseAttention over
// the kept blocks; the chain rule, the paper gives no backward) as one persistent,
// warp-specialised launch, for shifts that are multiples of 4, so that every window is one,
// two or four TMA boxes (window.cuh). The products, operand layouts and per-pair arithmetic are
// those of attn_bwd_tc.cu; what changes is who waits on what.
//
// Work items: a key block's dK, dV or a query block's dQ, of one (batch, head). The first item
// of a CTA is its index; the others come from a counter in the workspace that the row kernel
// zeroes. Key-block items come first (their lengths vary), query-block items fill in behind.
//   warp 11    producer: publishes each item (role, head, block, count and its list of other
//              blocks: the forward's list for dQ, the transposed list the row kernel built for
//              dK, dV) in one of two item slots; copies the item's resident tiles by TMA (two
//              buffers, by item parity) and each pair's streamed tiles (a ring of three), each
//              with the 512-byte row of (lse, D) values of its block that the compute warps
//              use (the row kernel writes them by block, in tile order: one bulk copy).
//   warps 8-10 lane 0 of each issues a share of the MMAs: warp 8 S and dK += dS^T Q, warp 9
//              dP and dV += P^T dO, warp 10 dQ += dS K. Per pair S, dP go into the same TMEM
//              columns once the compute warps hold the last ones in registers; the
//              accumulating products of a pair follow once its bf16 operands are stored.
//   warps 0-7  the exps and the bf16 operands of each pair, two warps per TMEM lane quadrant
//              (16 of a row's 64 columns a thread), and each item's epilogue (the accumulators
//              to global memory, fp32).
// Pairs are counted across items: the next item's tiles arrive while the last item computes,
// and its first products run while the compute warps store the last item's gradients.
// Tile rows follow the TMA box order (tile_row_pos). Every wait is bounded; on a timeout the
// CTA records SSBA_ERR_TIMEOUT, waits (bounded) for its copies and MMAs in flight, and returns.
#include <algorithm>
#include <cstdint>

#include "bwd_tile.cuh"
#include "common.cuh"
#include "ptx.cuh"
#include "window.cuh"

namespace ssba {

namespace {

using namespace ptx;
using namespace win;
using namespace bwd;

constexpr int kCompute = 256;   // warps 0-7, two per TMEM lane quadrant
constexpr int kIssuer0 = 256;   // lane 0 of warp 8: S, and dK += dS^T Q
constexpr int kIssuer1 = 288;   // lane 0 of warp 9: dP, and dV += P^T dO
constexpr int kIssuer2 = 320;   // lane 0 of warp 10: dQ += dS K
constexpr int kIssuers = 3;     // commit to bar_a, tile_empty, drain
constexpr int kSdpIssuers = 2;  // commit to bar_s, ab_empty
constexpr int kProducer = 11;   // warp
constexpr int kThreads = 384;
constexpr int kRing = 3;        // streamed tile slots
constexpr int kDone = -1;       // role of the item slot that ends a CTA's work
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColS = 0, kColDP = 64, kColA0 = 128, kColA1 = 192;
constexpr size_t kSmemBytes = 104 * 1024;  // two CTAs per SM (TMEM: 2 x 256 columns)

struct WsMaps {
    CUtensorMap q[4], k[4], v[4], o[4];  // Q, K, V, dO as window boxes (o: dO)
};

struct alignas(1024) WsSmem {
    uint8_t a[2][kTile];      // item tiles by item parity: dQ item Q_i, dK/dV item K_j
    uint8_t b[2][kTile];      //                            dO_i,         V_j
    uint8_t x[kRing][kTile];  // pair tiles: dQ item K_j, dK/dV item Q_i
    uint8_t y[kRing][kTile];  //             V_j,         dO_i
    uint8_t e[2][kTile];      // bf16 operands: dS (e[0]); P^T and dS^T
    float2 pld[kRing][kT];    // dK/dV pair: (lse log2(e), D) of its query rows (tile order)
    float2 ild[2][kT];        // dQ item: (lse log2(e), D) of its rows
    int list[2][256];         // the item's other blocks, in pair order (producer only)
    uint32_t win[256];        // label -> packed window entry (window_entry)
    int4 info[2];             // role (0 dQ, 1 dK/dV, kDone), bh, label, n
    uint64_t item_full[2];    // producer lane 0, after the slot is written
    uint64_t item_empty[2];   // the 8 compute warps and the 3 issuers have read the slot
    uint64_t ab_full[2];      // TMA bytes of the item tiles (and, for dQ, of its ild row)
    uint64_t ab_empty[2];     // MMA commits (the S and dP issuers) after the item's last S, dP
    uint64_t tile_full[kRing];   // TMA bytes of a pair's tiles (and, for dK/dV, of its pld row)
    uint64_t tile_empty[kRing];  // MMA commits (all three issuers) after the pair's products
    uint64_t bar_s;           // MMA commits (the S and dP issuers): S, dP of the pair in TMEM
    uint64_t s_free;          // 8 compute warps: S, dP in registers
    uint64_t e_full;          // 8 compute warps: the pair's bf16 operands stored
    uint64_t bar_a;           // MMA commits (all three issuers): the pair's accumulating products
    uint64_t drain;
    uint32_t tmem_base;
    int abort_flag;
};
static_assert(sizeof(WsSmem) + 1024 <= kSmemBytes, "shared memory");

__device__ __forceinline__ WsSmem& smem_layout()
{
    extern __shared__ uint8_t raw[];
    return *reinterpret_cast<WsSmem*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~static_cast<uintptr_t>(1023));
}

// A warp's bounded wait: every lane must see the phase, so a timeout takes the warp out whole.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abortf, uint64_t budget_ns)
{
    const bool ok = mbar_wait(bar, parity, abortf, budget_ns);
    return __all_sync(0xffffffffu, ok);
}

// One arrive per warp, after every lane's earlier TMEM loads and shared-memory writes.
__device__ __forceinline__ void warp_arrive(uint32_t bar)
{
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}

// Token of tile row r of block `label` (TMA box order).
__device__ __forceinline__ int tile_token(const Grid& g, int label, int r)
{
    return g.token(label, tile_row_pos(g, label, r));
}

constexpr uint32_t kLdRow = kT * sizeof(float2);  // 512 bytes of (lse, D) per block

// An item slot's shape, read after its mbarrier wait.
__device__ __forceinline__ int4 read_info(const int4* q)
{
    const volatile int* v = reinterpret_cast<const volatile int*>(q);
    return make_int4(v[0], v[1], v[2], v[3]);
}

// Item w: [0, nk) key blocks (role 1), then query blocks (role 0), bh-major.
__device__ __forceinline__ int4 decode_item(int w, int nk, int Tb)
{
    const bool key = w < nk;
    const int u = key ? w : w - nk, bh = u / Tb;
    return make_int4(key ? 1 : 0, bh, u - bh * Tb, 0);
}

// Warp 11. nk = number of key-block items (B * heads * Tb), total = 2 nk. Returns false on a
// timeout. P counts the pairs whose tiles were issued, kab the items whose tiles were issued
// (after a timeout the teardown waits for the last copies of each barrier).
__device__ bool produce(const WsMaps& maps, const BwdParams& p, WsSmem& sm, const int nk, uint32_t& P, int& kab)
{
    const int lane = threadIdx.x & 31;
    const Grid& g = p.g;
    const int Tb = g.Tb();
    volatile int* abortf = &sm.abort_flag;
    grid_dep_wait();  // D, the counter and the transposed lists come from the row kernel
    int w = blockIdx.x;
    kab = 0;
    for (int k = 0;; ++k) {
        const int s = k & 1;
        if (k >= 2 && !warp_wait(smem_u32(&sm.item_empty[s]), ((k >> 1) + 1) & 1, abortf, p.budget_ns))
            return false;
        if (w >= 2 * nk) {  // no work left: the end marker
            if (lane == 0) {
                sm.info[s] = make_int4(kDone, 0, 0, 0);
                mbar_arrive(smem_u32(&sm.item_full[s]));
            }
            return true;
        }
        const int4 it = decode_item(w, nk, Tb);
        const int role = it.x, bh = it.y, label = it.z;
        const size_t brow = (size_t)bh * Tb + label;
        int n;
        const int32_t* src;
        if (role == 1) {  // dK, dV: the query blocks whose lists hold this key block, ascending
            n = min(max(__ldg(p.tcnt + brow), 0), Tb);
            src = p.tlist + __ldg(p.toff + brow);
        } else {  // dQ: the forward's list
            n = min(max(__ldg(p.cnt + brow), 0), p.keep);
            src = p.idx + brow * p.keep;
        }
        for (int i = lane; i < n; i += 32) sm.list[s][i] = min(max(__ldg(src + i), 0), Tb - 1);
        __syncwarp();
        if (lane == 0) {
            sm.info[s] = make_int4(role, bh, label, n);
            mbar_arrive(smem_u32(&sm.item_full[s]));
        }
        // the item's resident tiles, once the item two back has issued its last S, dP
        if (k >= 2 && !warp_wait(smem_u32(&sm.ab_empty[s]), ((k >> 1) + 1) & 1, abortf, p.budget_ns)) return false;
        if (lane == 0) {
            const uint32_t bar = smem_u32(&sm.ab_full[s]), e = sm.win[label];
            mbar_arrive_expect_tx(bar, 2 * kTile + (role ? 0 : kLdRow));
            window_boxes_e(role ? maps.k : maps.q, smem_u32(sm.a[s]), bar, e, bh);
            window_boxes_e(role ? maps.v : maps.o, smem_u32(sm.b[s]), bar, e, bh);
            if (!role) bulk_load(smem_u32(sm.ild[s]), p.ld + brow * kT, kLdRow, bar);
        }
        ++kab;
        // the pairs' streamed tiles, each once the pair three back has finished its products
        for (int t = 0; t < n; ++t, ++P) {
            const int r = (int)(P % kRing);
            if (P >= kRing && !warp_wait(smem_u32(&sm.tile_empty[r]), ((P / kRing) + 1) & 1, abortf, p.budget_ns))
                return false;
            const int j = sm.list[s][t];
            // test hook: CTA 0 announces its first pair's bytes and copies nothing, so that the
            // waits on them run out
            const bool hold = p.withhold == 1 && P == 0 && blockIdx.x == 0;
            if (lane == 0) {
                const uint32_t bar = smem_u32(&sm.tile_full[r]), e = sm.win[j];
                mbar_arrive_expect_tx(bar, 2 * kTile + (role ? kLdRow : 0));
                if (!hold) {
                    window_boxes_e(role ? maps.q : maps.k, smem_u32(sm.x[r]), bar, e, bh);
                    window_boxes_e(role ? maps.o : maps.v, smem_u32(sm.y[r]), bar, e, bh);
                    if (role) bulk_load(smem_u32(sm.pld[r]), p.ld + ((size_t)bh * Tb + j) * kT, kLdRow, bar);
                }
            }
        }
        int next = 0;
        if (lane == 0) next = (int)gridDim.x + atomicAdd(p.ctr, 1);
        w = __shfl_sync(0xffffffffu, next, 0);
    }
}

// Issuer `which`'s share of the accumulating products of pair q (its role, and whether it opens
// its item), once the pair's bf16 operands are stored: for a key-block pair issuer 0
// dK += dS^T Q (x tile), issuer 1 dV += P^T dO (y tile); nothing for a query-block pair, whose
// dQ is issuer 2's. Each commits, so bar_a and tile_empty count three.
__device__ __forceinline__ bool issue_acc(const BwdParams& p, WsSmem& sm, uint32_t q, int role, bool first, int which)
{
    if (!mbar_wait(smem_u32(&sm.e_full), q & 1, &sm.abort_flag, p.budget_ns)) return false;
    tc_fence_after();
    const uint32_t tb0 = sm.tmem_base;
    const int r = (int)(q % kRing);
    if (role == 1) {
        if (which == 0)
            mma_sb(tb0 + kColA1, smem_u32(sm.e[1]), smem_u32(sm.x[r]), !first);  // dK += dS^T Q
        else
            mma_sb(tb0 + kColA0, smem_u32(sm.e[0]), smem_u32(sm.y[r]), !first);  // dV += P^T dO
    }
    mma_commit(smem_u32(&sm.bar_a));
    mma_commit(smem_u32(&sm.tile_empty[r]));
    return true;
}

// Lane 0 of warp 8 (which = 0) or 9 (which = 1): S or dP of every pair and its share of the
// accumulating products, so that the issue latency of a tcgen05.mma (about 57 cycles from one
// thread, 44 a product when several issue) is shared. Returns false on a timeout.
// Lane 0 of warp 10: dQ += dS K of every query-block pair, in pair order, once its operands are
// stored; for key-block pairs it only commits (bar_a and tile_empty count three commits).
__device__ bool issue_dq(const BwdParams& p, WsSmem& sm)
{
    volatile int* abortf = &sm.abort_flag;
    const uint32_t tb0 = sm.tmem_base;
    uint32_t P = 0;
    for (int k = 0;; ++k) {
        const int s = k & 1;
        if (!mbar_wait(smem_u32(&sm.item_full[s]), (k >> 1) & 1, abortf, p.budget_ns)) return false;
        const int4 inf = read_info(&sm.info[s]);
        mbar_arrive(smem_u32(&sm.item_empty[s]));
        if (inf.x == kDone) return true;
        const int role = inf.x, n = inf.w;
        for (int t = 0; t < n; ++t, ++P) {
            if (!mbar_wait(smem_u32(&sm.e_full), P & 1, abortf, p.budget_ns)) return false;
            tc_fence_after();
            const int r = (int)(P % kRing);
            if (role == 0) mma_sb(tb0 + kColA0, smem_u32(sm.e[0]), smem_u32(sm.x[r]), t > 0);  // dQ += dS K
            mma_commit(smem_u32(&sm.bar_a));
            mma_commit(smem_u32(&sm.tile_empty[r]));
        }
    }
}

__device__ bool issue(const BwdParams& p, WsSmem& sm, const int which)
{
    volatile int* abortf = &sm.abort_flag;
    const uint32_t tb0 = sm.tmem_base;
    uint32_t P = 0;  // pairs whose S, dP are issued
    bool pending = false;  // pair P - 1's accumulating products not yet issued
    int prole = 0;
    bool pfirst = false;
    for (int k = 0;; ++k) {
        const int s = k & 1;
        // the last item's final products first: its epilogue waits for them, and the next
        // item's tiles may still be on their way
        if (pending) {
            if (!issue_acc(p, sm, P - 1, prole, pfirst, which)) return false;
            pending = false;
        }
        if (!mbar_wait(smem_u32(&sm.item_full[s]), (k >> 1) & 1, abortf, p.budget_ns)) return false;
        const int4 inf = read_info(&sm.info[s]);
        mbar_arrive(smem_u32(&sm.item_empty[s]));
        if (inf.x == kDone) return true;
        const int role = inf.x, n = inf.w;
        if (!mbar_wait(smem_u32(&sm.ab_full[s]), (k >> 1) & 1, abortf, p.budget_ns)) return false;
        const uint32_t ab = smem_u32(which ? sm.b[s] : sm.a[s]);
        for (int t = 0; t < n; ++t, ++P) {
            const int r = (int)(P % kRing);
            if (!mbar_wait(smem_u32(&sm.tile_full[r]), (P / kRing) & 1, abortf, p.budget_ns)) return false;
            if (P > 0 && !mbar_wait(smem_u32(&sm.s_free), (P - 1) & 1, abortf, p.budget_ns)) return false;
            tc_fence_after();
            if (which == 0)
                mma_kk(tb0 + kColS, ab, smem_u32(sm.x[r]));  // S = Q K^T (dK/dV item: S^T = K Q^T)
            else
                mma_kk(tb0 + kColDP, ab, smem_u32(sm.y[r]));  // dP = dO V^T (dP^T = V dO^T)
            mma_commit(smem_u32(&sm.bar_s));
            if (t == n - 1) mma_commit(smem_u32(&sm.ab_empty[s]));
            if (pending && !issue_acc(p, sm, P - 1, prole, pfirst, which)) return false;
            pending = true;
            prole = role;
            pfirst = t == 0;
        }
        if (n == 0) mma_commit(smem_u32(&sm.ab_empty[s]));
    }
}

// Columns [col0, col0 + 16) of this thread's row of the fp32 accumulator whose 16-column
// group starts at TMEM address taddr, times mul, to row `token` of out (one [N][64] head).
__device__ __forceinline__ void store_cols(uint32_t taddr, float* out, int token, int col0, float mul)
{
    uint32_t v[16];
    tmem_ld_16x32bx2_x16_off32(taddr, v);
    tmem_wait_ld();
    float4* dst = reinterpret_cast<float4*>(out + (size_t)token * kD + col0);
#pragma unroll
    for (int i = 0; i < 4; ++i)
        dst[i] = make_float4(__uint_as_float(v[4 * i]) * mul, __uint_as_float(v[4 * i + 1]) * mul,
                             __uint_as_float(v[4 * i + 2]) * mul, __uint_as_float(v[4 * i + 3]) * mul);
}

// Sixteen bf16 values (8 packed pairs) of row r, 16-byte chunks c0 and c0 + 1, into the
// 128-byte-swizzled K-major tile at dst.
__device__ __forceinline__ void store_cols_bf16(uint8_t* dst, int r, int c0, const uint32_t (&v)[8])
{
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int c = c0 + i;
        *reinterpret_cast<uint4*>(dst + r * 128 + ((c ^ (r & 7)) << 4)) =
            make_uint4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
    }
}

// Warps 0-7: warp w reads TMEM lane quadrant w % 4; thread (w, lane) owns row
// r = 16 (w % 4) + lane % 16 of the M=64 data path and its columns [col0, col0 + 16),
// col0 = 32 (lane / 16) + 16 (w / 4): two warps share each quadrant's exps. Returns false on a
// timeout.
__device__ bool compute(const BwdParams& p, WsSmem& sm)
{
    volatile int* abortf = &sm.abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int q = warp & 3, col0 = 32 * (lane >> 4) + 16 * (warp >> 2);
    const int r = q * 16 + (lane & 15);
    // lanes 16-31 of a 16x32bx2 load read 32 columns further on: one address serves the warp
    const uint32_t tb = sm.tmem_base + (static_cast<uint32_t>(q * 32) << 16) + 16 * (warp >> 2);
    const Grid& g = p.g;
    const int N = g.H * g.W;
    const float c = p.scale * kLog2e;
    uint32_t P = 0;  // pairs done
    for (int k = 0;; ++k) {
        const int s = k & 1;
        if (!warp_wait(smem_u32(&sm.item_full[s]), (k >> 1) & 1, abortf, p.budget_ns)) return false;
        const int4 inf = read_info(&sm.info[s]);
        float L2 = 0.f, Dr = 0.f;
        if (inf.x == 0) {  // the row's statistics came with the item's tiles
            if (!warp_wait(smem_u32(&sm.ab_full[s]), (k >> 1) & 1, abortf, p.budget_ns)) return false;
            L2 = sm.ild[s][r].x;
            Dr = sm.ild[s][r].y;
        }
        warp_arrive(smem_u32(&sm.item_empty[s]));
        if (inf.x == kDone) return true;
        const int role = inf.x, bh = inf.y, label = inf.z, n = inf.w;
        for (int t = 0; t < n; ++t, ++P) {
            const int slot = (int)(P % kRing);
            if (!warp_wait(smem_u32(&sm.bar_s), P & 1, abortf, p.budget_ns)) return false;
            tc_fence_after();
            uint32_t sv[16], dp[16];
            tmem_ld_16x32bx2_x16_off32(tb + kColS, sv);
            tmem_ld_16x32bx2_x16_off32(tb + kColDP, dp);
            tmem_wait_ld();
            tc_fence_before();
            warp_arrive(smem_u32(&sm.s_free));
            if (role == 1) {
                // S^T, dP^T: columns are the query rows col0 + i of the pair's query block
                if (!warp_wait(smem_u32(&sm.tile_full[slot]), (P / kRing) & 1, abortf, p.budget_ns)) return false;
                const float4* ld = reinterpret_cast<const float4*>(sm.pld[slot] + col0);
                uint32_t pp[8], dd[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float4 qd = ld[i];  // (lse, D) of query rows col0 + 2 i and col0 + 2 i + 1
                    const float p0 = fast_exp2(fmaf(__uint_as_float(sv[2 * i]), c, -qd.x));
                    const float p1 = fast_exp2(fmaf(__uint_as_float(sv[2 * i + 1]), c, -qd.z));
                    pp[i] = pack_bf16(p0, p1);
                    dd[i] = pack_bf16(p0 * (__uint_as_float(dp[2 * i]) - qd.y), p1 * (__uint_as_float(dp[2 * i + 1]) - qd.w));
                }
                // the last pair's products have read e[] (and the tiles of its slot)
                if (P > 0 && !warp_wait(smem_u32(&sm.bar_a), (P - 1) & 1, abortf, p.budget_ns)) return false;
                store_cols_bf16(sm.e[0], r, col0 >> 3, pp);
                store_cols_bf16(sm.e[1], r, col0 >> 3, dd);
            } else {
                uint32_t pk[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float p0 = fast_exp2(fmaf(__uint_as_float(sv[2 * i]), c, -L2));
                    const float p1 = fast_exp2(fmaf(__uint_as_float(sv[2 * i + 1]), c, -L2));
                    pk[i] = pack_bf16(p0 * (__uint_as_float(dp[2 * i]) - Dr), p1 * (__uint_as_float(dp[2 * i + 1]) - Dr));
                }
                if (P > 0 && !warp_wait(smem_u32(&sm.bar_a), (P - 1) & 1, abortf, p.budget_ns)) return false;
                store_cols_bf16(sm.e[0], r, col0 >> 3, pk);
            }
            fence_proxy_async_smem();
            warp_arrive(smem_u32(&sm.e_full));
        }
        // epilogue: the item's gradients, rows in tile order
        const size_t head = (size_t)bh * N * kD;
        const int tok = tile_token(g, label, r);
        if (n > 0) {
            if (!warp_wait(smem_u32(&sm.bar_a), (P - 1) & 1, abortf, p.budget_ns)) return false;
            tc_fence_after();
            if (role == 1) {
                store_cols(tb + kColA0, p.dV + head, tok, col0, 1.0f);
                store_cols(tb + kColA1, p.dK + head, tok, col0, p.scale);
            } else {
                store_cols(tb + kColA0, p.dQ + head, tok, col0, p.scale);
            }
            tc_fence_before();  // the next item's first products overwrite the accumulators
        } else {
            float4* a = reinterpret_cast<float4*>((role == 1 ? p.dV : p.dQ) + head + (size_t)tok * kD + col0);
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (role == 1) {
                float4* b = reinterpret_cast<float4*>(p.dK + head + (size_t)tok * kD + col0);
#pragma unroll
                for (int i = 0; i < 4; ++i) b[i] = make_float4(0.f, 0.f, 0.f, 0.f);
            }
        }
    }
}

__global__ void __launch_bounds__(kThreads, 2) ssba_bwd_ws_kernel(const __grid_constant__ WsMaps maps, const BwdParams p,
                                                               const int nk)
{
    WsSmem& sm = smem_layout();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        sm.abort_flag = 0;
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&sm.item_full[i]), 1);
            mbar_init(smem_u32(&sm.item_empty[i]), kCompute / 32 + kIssuers);
            mbar_init(smem_u32(&sm.ab_full[i]), 1);
            mbar_init(smem_u32(&sm.ab_empty[i]), kSdpIssuers);
        }
        for (int i = 0; i < kRing; ++i) {
            mbar_init(smem_u32(&sm.tile_full[i]), 1);
            mbar_init(smem_u32(&sm.tile_empty[i]), kIssuers);
        }
        mbar_init(smem_u32(&sm.bar_s), kSdpIssuers);
        mbar_init(smem_u32(&sm.s_free), kCompute / 32);
        mbar_init(smem_u32(&sm.e_full), kCompute / 32);
        mbar_init(smem_u32(&sm.bar_a), kIssuers);
        mbar_init(smem_u32(&sm.drain), kIssuers);
        fence_mbar_init();
    }
    for (int l = threadIdx.x; l < p.g.Tb(); l += kThreads) sm.win[l] = window_entry(p.g, l);
    if (warp == kProducer && lane < 16) {
        const CUtensorMap* m = lane < 4 ? &maps.q[lane] : lane < 8 ? &maps.k[lane - 4] : lane < 12 ? &maps.v[lane - 8]
                                                                                                  : &maps.o[lane - 12];
        tma_prefetch_desc(m);
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(&sm.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    bool ok = true;
    uint32_t P = 0;
    int kab = 0;
    if (warp < kCompute / 32)
        ok = compute(p, sm);
    else if (threadIdx.x == kIssuer0 || threadIdx.x == kIssuer1)
        ok = issue(p, sm, threadIdx.x == kIssuer1 ? 1 : 0);
    else if (threadIdx.x == kIssuer2)
        ok = issue_dq(p, sm);
    else if (warp == kProducer)
        ok = produce(maps, p, sm, nk, P, kab);
    const bool dead = __syncthreads_or(!ok);

    if (dead) {  // nothing more is issued: wait (bounded) for what is in flight, then report
        volatile int* abortf = &sm.abort_flag;
        *abortf = 1;
        if (warp == kProducer && lane == 0) {
            const uint64_t t0 = globaltimer_ns();
            auto settle = [&](uint32_t bar, uint32_t parity) {
                while (!mbar_try_wait(bar, parity) && globaltimer_ns() - t0 < p.budget_ns) {
                }
            };
            for (int i = 1; i <= 2 && i <= kab; ++i) settle(smem_u32(&sm.ab_full[(kab - i) & 1]), ((kab - i) >> 1) & 1);
            for (uint32_t i = 1; i <= (uint32_t)kRing && i <= P; ++i) {
                const uint32_t q = P - i;
                settle(smem_u32(&sm.tile_full[q % kRing]), (q / kRing) & 1);
            }
        }
        if (threadIdx.x == kIssuer0 || threadIdx.x == kIssuer1 || threadIdx.x == kIssuer2) {  // drain counts 3
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
    if (warp == 0) tmem_dealloc(sm.tmem_base, kTmemCols);
}

}  // namespace

int launch_backward_ws(const ssba_desc& d, const Grid& g, int keep, float scale, const void* Q, const void* K,
                       const void* V, const void* O, const float* lse, const void* dO, const int32_t* idx,
                       const int32_t* cnt, float* dQ, float* dK, float* dV, void* workspace, cudaStream_t st,
                       uint64_t budget_ns, int withhold)
{
    if (d.head_dim != kD || g.blk != 8 || d.dtype != SSBA_BF16 || g.Tb() > 256 || (g.sr % 4) || (g.sc % 4))
        return SSBA_ERR_UNSUPPORTED;
    const int BH = d.B * d.heads;
    WsMaps maps;
    if (!encode_window_maps(maps.q, Q, BH, g.H, g.W) || !encode_window_maps(maps.k, K, BH, g.H, g.W) ||
        !encode_window_maps(maps.v, V, BH, g.H, g.W) || !encode_window_maps(maps.o, dO, BH, g.H, g.W))
        return SSBA_ERR_UNSUPPORTED;  // e.g. a base address the tensor maps cannot take
    const BwdLayout lay = bwd_layout(d, g, keep);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
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
    p.Dbuf = reinterpret_cast<float*>(ws);
    p.ctr = reinterpret_cast<int*>(ws + lay.ctr);
    p.toff = reinterpret_cast<int*>(ws + lay.toff);
    p.tcnt = reinterpret_cast<int*>(ws + lay.tcnt);
    p.tlist = reinterpret_cast<int*>(ws + lay.tlist);
    p.ld = reinterpret_cast<float2*>(ws + lay.ld);
    p.g = g;
    p.keep = keep;
    p.scale = scale;
    p.budget_ns = budget_ns;
    p.withhold = withhold;
    p.status = device_status_word();
    if (!p.status) {
        set_error("ssba_backward: could not resolve the device status word");
        return SSBA_ERR_CUDA;
    }
    static PerDeviceOnce attr;
    attr.run([] {
        cudaFuncSetAttribute(ssba_bwd_ws_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    });
    cudaError_t e = launch_bwd_rows(p, BH, st);
    if (e == cudaSuccess) {
        const int nk = BH * g.Tb();
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)std::min(2 * device_sm_count(), 2 * nk));
        cfg.blockDim = dim3(kThreads);
        cfg.dynamicSmemBytes = kSmemBytes;
        cfg.stream = st;
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        at[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, ssba_bwd_ws_kernel, maps, p, nk);
    }
    if (e != cudaSuccess) {
        set_error("ssba_backward (persistent tensor-core kernel) launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

}  // namespace ssba
