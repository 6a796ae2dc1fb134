// attn_tc.cu -- bf16 block-sparse attention forward on the sm_103a tensor cores
// (Sec. 2.2 "Efficient Sparse Execution": the kernel skips pruned blocks in its loads
// and its MMAs; Algorithm 1 SparseAttention over image tokens).
//
// Work item = one query block (64 tokens, an 8x8 window of the shifted grid) of one
// (batch, head); it visits only the key blocks listed for it. Persistent CTAs, one per SM
// (its 205 KB of shared memory fills the SM), each running two independent
// pipelines of 12 warps (768 threads), warp-specialised by warpgroup:
//   warp 0      TMA producer (Q, K). Q of each item and K, V of each listed key block arrive as
//               8 KB tiles cut from [B*heads, H, W, d] tensor maps (128-byte swizzle): one
//               8x8-token box when the shifted window does not cross the grid edge, else two
//               or four boxes. A half-block shift is a multiple of 4 tokens, so a crossing
//               window splits 4 + 4: no gather pass and no out-of-range fill. Q is
//               double-buffered; K and V have separate 5-stage rings (a K slot frees when
//               its QK is done, a V slot when its PV is done).
//   warp 1      QK issuer (one elected lane; warp 1 of the CTA also owns the TMEM allocation):
//                 S_t = Q K_t^T   tcgen05.mma kind::f16, M=64 N=64, A = Q tile and
//                                 B = K tile from shared memory (K-major, SW128)
//               S is triple-buffered in TMEM: QK of block t waits only until PV_{t-3} has
//               read P_{t-3} from the same buffer.
//   warp 2      TMA producer of the V ring (warp 0 keeps Q and K), so that two threads
//               share the per-box issue latency.
//   warp 3      PV issuer (one elected lane):
//                 O  += P_t V_t   tcgen05.mma kind::f16, M=64 N=64, A = P from TMEM,
//                                 B = V tile (MN-major, SW128)
//               P_t (bf16 pairs, 32 columns) goes into the first half of S_t's buffer, which
//               the softmax no longer needs once S_t is in its registers, so the softmax never
//               waits for a P buffer and QK runs up to three blocks ahead. TMEM of a
//               pipeline: S/P 3 x 64 + O 64 = 256 columns. Two issuing threads keep one's
//               barrier waits (about 100 cycles per query) off the other's issue path.
//   warps 4-7   softmax, one TMEM lane quadrant each. The M=64 data path puts tile row r
//               at lane 32*(r/16) + r%16, so two threads share a row (16x32bx2 TMEM
//               loads), each holding 32 of its 64 scores. Online softmax in fp32 with exp2
//               in the log2-scaled domain; the running max is only raised when it grows by
//               more than 2^8, which keeps P <= 256 in bf16; O is then rescaled in TMEM
//               after P_t is stored, so that S and O never share the registers (80 per
//               thread: 768 threads on one SM). At the end of an item the row statistics
//               (max, sum) go to shared memory.
//   warps 8-11  epilogue: O / l in bf16 and lse, overlapping the next item's softmax.
// In-kernel selection (ssba_forward_select): given the block means, each CTA first computes
// the score rows and the Top-k gating of its own items (one warp per item, the arithmetic of
// the mask kernels) and writes the lists to the caller's kv_idx / kv_cnt, which its producers
// then read back (coherent loads); no separate selection launch and no cross-CTA dependency.
// Tile rows follow the TMA box order of the window (tile_row_pos). All mbarrier waits are
// bounded (globaltimer budget + CTA abort flag); a timeout is reported in the device status
// word and the CTA drains its in-flight copies and MMAs before it exits.
#include <cuda.h>
#include <cstdio>
#include <cstring>

#include "common.cuh"
#include "ptx.cuh"
#include "select.cuh"
#include "window.cuh"

namespace ssba {

namespace {

using namespace ptx;
using namespace win;

constexpr int kD = 64;
constexpr int kRows = 64;  // query rows per item = tokens per block
constexpr int kKStages = 5;  // K ring
constexpr int kVStages = 5;  // V ring
constexpr int kSBuf = 3;     // S buffers in TMEM (fp32, 64 columns each); P_t (bf16 pairs) goes
                             // into the first 32 columns of S_t's buffer
constexpr int kSlotWarps = 12;                // warps of one pipeline (see the role map above)
constexpr int kSlots = 2;                     // independent pipelines per CTA
constexpr int kThreads = kSlots * kSlotWarps * 32;
constexpr uint32_t kSlotCols = 256;           // TMEM columns of one pipeline
constexpr uint32_t kTmemCols = kSlots * kSlotCols;
constexpr uint32_t kColS = 0;    // S / P buffers: [0,64), [64,128), [128,192)
constexpr uint32_t kColO = 192;  // O accumulator: [192,256)
constexpr uint32_t kTileBytes = kRows * kD * 2;  // 8 KB
constexpr float kRescaleLog2 = 8.0f;
constexpr int kLabelCap = 128;  // labels staged per producer warp and piece; the rest are read per block
constexpr int kCntCap = 64;     // phase-B item counts of a pipeline held in shared memory
constexpr int kCntA = 3;        // phase-A pieces of one pipeline: at most three
constexpr int kSplitMinKeep = 24;  // shortest list for which items are cut to balance the pipelines

// QK: M=64 N=64, A (Q) and B (K) K-major. PV: M=64 N=64, A (P) K-major, B (V) MN-major.
constexpr uint32_t kIdescQK = idesc_bf16_f32(64, 64, false, false);
constexpr uint32_t kIdescPV = idesc_bf16_f32(64, 64, false, true);

struct __align__(1024) SlotSmem {
    uint8_t k[kKStages][kTileBytes];
    uint8_t v[kVStages][kTileBytes];
    uint8_t q[2][kTileBytes];
    float2 stats[2][kRows];  // (max in log2 units, row sum) per item parity
    uint64_t k_full[kKStages];
    uint64_t k_empty[kKStages];
    uint64_t v_full[kVStages];
    uint64_t v_empty[kVStages];
    uint64_t q_full[2];
    uint64_t q_empty[2];
    uint64_t s_full[kSBuf];
    uint64_t s_free[kSBuf];   // PV_t has finished (it read P_t from S_t's buffer): QK_{t+3} may
                              // overwrite the buffer
    uint64_t p_full[kSBuf];
    uint64_t stats_full[2];
    uint64_t stats_free[2];
    uint64_t o_full;
    uint64_t o_free;
    uint64_t drain[2];
    int32_t labels[2][kLabelCap];     // [producer warp] key-block labels of the current piece
    int32_t cnts[kCntCap];            // counts of the first phase-B items, in walk order
    int4 pieceA[kCntA];               // phase-A pieces in walk order: item, tb, nb, part
    int nA, nB, M;                    // phase-A pieces, phase-B items, phase-A items (all pipelines)
};

constexpr int kWinCap = 256;  // labels whose window (origin, box shape) is tabulated per CTA (2048 px: 256)

// Timeline instrumentation, compiled only into the timeline build of the library (-DSSBA_TIMELINE;
// the default build has none of it). Per CTA, globaltimer stamps (ns) of the launch's phases; per
// tile of eight sampled pipelines (pipeline 0 and 1 of CTAs 0, 1, gridDim/2 and gridDim-1), SM
// clock stamps of each role's step, and per item the epilogue's. ssba_timeline_read copies them out.
namespace tl {
constexpr int kCtas = 256, kCtaEv = 16, kPipes = 4 * kSlots, kTiles = 128, kTileEv = 12, kItems = 32, kItemEv = 4;
enum CtaEv { kEntry = 0, kDepWait, kPoolLanded, kPooled, kBarrier, kStaged, kSelected, kPipesStart, kSlot0End,
             kSlot1End, kEnd, kSelStart, kScoresDone, kWalkDone };
// tile events: K copy issued, QK issued, softmax saw S, softmax done with the exps, P stored,
// PV issued, V copy issued, QK's wait for a free S buffer over, S in the softmax's registers,
// row maxima known, P buffer free (softmax), PV's waits over
enum TileEv { kKIssue = 0, kQKIssue, kSmxStart, kSmxExp, kPStored, kPVIssue, kVIssue, kSFree, kSLoaded, kMaxDone,
              kPFree, kPVReady };
enum ItemEv { kEpiStart = 0, kEpiO, kEpiDone, kPipeClock0 };
#ifdef SSBA_TIMELINE
__device__ unsigned long long cta_ev[kCtas][kCtaEv];
__device__ unsigned int tile_ev[kPipes][kTiles][kTileEv];
__device__ unsigned int item_ev[kPipes][kItems][kItemEv];
__device__ __forceinline__ int pipe_of(int slot)
{
    const int b = blockIdx.x, G = gridDim.x;
    const int s = b == 0 ? 0 : (b == 1 ? 1 : (b == G / 2 ? 2 : (b == G - 1 ? 3 : -1)));
    return s < 0 ? -1 : s * kSlots + slot;
}
#endif
}  // namespace tl
// -DSSBA_TIMELINE=1 records the per-CTA phase stamps only (they barely perturb the launch);
// -DSSBA_TIMELINE=2 also the per-tile and per-item stamps of the sampled pipelines.
#ifdef SSBA_TIMELINE
#define TL_CTA(ev)                                                                              \
    do {                                                                                        \
        if (blockIdx.x < tl::kCtas) tl::cta_ev[blockIdx.x][ev] = ptx::globaltimer_ns();        \
    } while (0)
#if SSBA_TIMELINE >= 2
#define TL_TILE(slot, gb, ev)                                                                   \
    do {                                                                                        \
        const int tl_p_ = tl::pipe_of(slot);                                                    \
        if (tl_p_ >= 0 && (gb) < (uint32_t)tl::kTiles) tl::tile_ev[tl_p_][gb][ev] = (unsigned)clock(); \
    } while (0)
#define TL_ITEM(slot, n, ev)                                                                    \
    do {                                                                                        \
        const int tl_p_ = tl::pipe_of(slot);                                                    \
        if (tl_p_ >= 0 && (n) < (uint32_t)tl::kItems) tl::item_ev[tl_p_][n][ev] = (unsigned)clock(); \
    } while (0)
#else
#define TL_TILE(slot, gb, ev) do { } while (0)
#define TL_ITEM(slot, n, ev) do { } while (0)
#endif
#else
#define TL_CTA(ev) do { } while (0)
#define TL_TILE(slot, gb, ev) do { } while (0)
#define TL_ITEM(slot, n, ev) do { } while (0)
#endif

struct __align__(1024) SmemLayout {
    SlotSmem slot[kSlots];
    uint32_t win[kWinCap];  // label -> r0 | c0 << 15 | box shape << 30 (see window_entry)
    uint64_t pool_bar[kThreads / 32];  // one per warp: its block's rows landed (in-kernel pooling)
    uint32_t tmem_base;
    int abort_flag;
};

// Four maps per tensor, one per box shape, over the [B*heads][H][W][d] bf16 view, and
// the text keys and values as [B*heads][T_txt][d] (64-row boxes, zero fill past T_txt).
static_assert(sizeof(SmemLayout) + 1024 <= 232448, "shared memory of one CTA (227 KB opt-in limit)");

struct TileMaps {
    CUtensorMap q[4], k[4], v[4];
    CUtensorMap kt, vt;
};

struct TcParams {
    __nv_bfloat16* O;
    float* lse;
    const int32_t* idx;  // null: dense mode, every block of the head
    const int32_t* cnt;
    Grid g;
    int keep;          // length of an index-list row
    int ntxt;          // text key blocks visited first by every query block (ceil(T_txt / 64))
    int t_txt;         // text tokens
    int units;         // key blocks of a whole item: ntxt + keep
    int num_items;
    float scale_log2;  // softmax scale * log2(e)
    int* status;       // device status word
    // Split-merge workspace (null when the caller gave none; then split = 0).
    int split;         // 1: pipelines take equal ranges of blocks, items may be cut in two
    int* ws_cnt;       // [boundaries][4] arrival counters, zero between launches
    float2* ws_st;     // [boundaries][2][64] row (max in log2 units, sum) of each part
    float* ws_o;       // [boundaries][2][64][64] unnormalised O of each part, fp32
    const float* sel_qb;  // in-kernel selection: block means [B*heads][Tb][64] (null: lists given)
    const float* sel_kb;
    int32_t* sel_cnt;     // counts written by the selection
    float* sel_scores;    // optional S export [B*heads][Tb][Tb]
    // in-kernel pooling (ssba_forward_fused): every warp of the grid pools one (block, tensor)
    // unit into sel_qb / sel_kb, then the CTAs meet at a grid barrier (null: means given)
    const __nv_bfloat16* pool_q;
    const __nv_bfloat16* pool_k;
    unsigned* gsync;  // grid barrier words in the workspace (arrivals, departures)
    uint64_t budget_ns;  // wall-time limit of every barrier wait
    int withhold;        // failure-detection test hooks: 1, pipeline 0 announces its first K copy
                         // but never issues it, so that the waits on it run out; 2, CTA 0 does not
                         // arrive at the grid barrier of the fused launch (0 otherwise)
};

// Work schedule, for V pipelines (two per CTA).
//   split = 0: whole items round-robin, item v + r V for pipeline v (neighbouring pipelines
//     work on neighbouring items, so the K/V tiles of a few heads are shared through L2).
//   split = 1 (a workspace was given and items is not a multiple of V, items >= V): the
//     first M = items - (floor(items / V) - 1) V items (V <= M < 2V) form phase A, the rest
//     phase B. Phase A counts in units (item, key block), item u / keep, block u % keep (a
//     block past the item's count is an empty unit); pipeline v takes the units
//     [floor(M keep v / V), floor(M keep (v+1) / V)), at least keep of them, so an item is
//     cut at most once: at boundary v, into a first part (the last item of pipeline v-1)
//     and a second part (the first item of pipeline v). Each part writes its unnormalised
//     O and row statistics to the workspace, and the part that arrives second at the
//     boundary's counter merges the two (two partial softmax sums combine by rescaling
//     each by 2^(m_part - m), m the larger maximum, and adding) and resets the counter.
//     Phase B is whole items round-robin, item M + v + r V. Every pipeline then has the
//     same number of key blocks, give or take one.
// A pipeline runs phase A first and, in it, its cut last item first, so that both parts
// of every cut item finish early and the merges (a few global-memory round trips)
// overlap later work instead of lengthening the end of the kernel.
// Under in-kernel selection the items go to the pipelines in contiguous ranges (item counts
// differing by at most one), so that the few items of a CTA share one or two heads and the
// selection stages each head's k_b once.
__device__ __forceinline__ int sel_item_count(const TcParams& p, int v, int V)
{
    return p.num_items / V + (v < p.num_items % V ? 1 : 0);
}
__device__ __forceinline__ int sel_first_item(const TcParams& p, int v, int V)
{
    return v * (p.num_items / V) + min(v, p.num_items % V);
}

__device__ __forceinline__ int split_items(const TcParams& p, int V)
{
    return p.split ? p.num_items - (p.num_items / V - 1) * V : 0;
}

struct Piece {
    int item;  // (batch, head) * Tb + query-block label
    int tb;    // first block (position in the item's list)
    int nb;    // blocks of this piece (0 for an empty piece)
    int part;  // -1 whole item, 0 first part (boundary v + 1), 1 second part (boundary v)
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
    uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity))
        if (globaltimer_ns() - t0 > budget_ns) return false;
    return true;
}

// 16x32bx2 store of 16 fp32 columns, threads 16-31 at +32 columns (counterpart of
// tmem_ld_16x32bx2_x16_off32), used for the O rescale.
__device__ __forceinline__ void tmem_st_16x32bx2_x16_off32(uint32_t taddr, const uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.16x32bx2.x16.b32 [%0], 32, "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
        "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}

__device__ __forceinline__ int clamp_label(int j, int Tb) { return j < 0 ? 0 : (j >= Tb ? Tb - 1 : j); }

// Checked build (-DSSBA_CHECKED, build.py variant "checked"): the invariants of the index lists
// the kernel reads (every label in [0, Tb), each row strictly ascending, every count in [0, keep])
// are tested, and a violation is reported as SSBA_ERR_CHECK in the device status word; the value
// is still clamped as in the default build, which tests nothing.
#ifdef SSBA_CHECKED
constexpr bool kChecked = true;
#else
constexpr bool kChecked = false;
#endif

// Block means of the whole layer inside the launch: unit u is (tensor u & 1, item u >> 1), one
// unit per warp and round, assigned warp-major over the grid so that the CTAs get equal
// shares. Lanes 0..7 bulk-copy the unit's eight token rows (one copy per row, two where the
// shifted window wraps the right edge) into this warp's 8 KB of the idle stage buffers, and
// after the copies land every lane sums its (row group, column chunk) with the loop order of
// ssba_pool_blocks_kernel, so the means are those of ssba_pool_blocks bit for bit. Returns
// false if a copy did not land in time (after a second bounded wait for it).
__device__ __noinline__ bool pool_phase(const TcParams& p, SmemLayout& cs, int gwarp, int lane, volatile int* abortf)
{
    constexpr int VE = 8, CPR = kD / VE, RPI = 32 / CPR, LOADS = 64 / RPI;
    constexpr int kWarps = kThreads / 32, kPerSlot = kWarps / kSlots;
    static_assert(kPerSlot * kTileBytes <= (kKStages + kVStages + 2) * kTileBytes, "pool buffers");
    const Grid& g = p.g;
    const int Tb = g.Tb(), N = g.H * g.W;
    const int col = lane % CPR, r0 = lane / CPR;
    const uint8_t* buf = &cs.slot[gwarp / kPerSlot].k[0][0] + (gwarp % kPerSlot) * kTileBytes;
    const uint32_t bar = smem_u32(&cs.pool_bar[gwarp]);
    const int nw = gridDim.x * kWarps;
    int round = 0;
    for (int u = gwarp * gridDim.x + blockIdx.x; u < 2 * p.num_items; u += nw, ++round) {
        const int which = u & 1, item = u >> 1;
        const int bh = item / Tb, label = item - bh * Tb;
        const int br = label / g.bw, bc = label - br * g.bw;
        const int rb = br * 8 - g.sr, cb = bc * 8 - g.sc;
        if (round > 0) {
            __syncwarp();
            fence_proxy_async_smem();  // the last round's reads before the copies overwrite them
        }
        if (lane == 0) mbar_arrive_expect_tx(bar, kTileBytes);
        __syncwarp();
        if (lane < 8) {
            const __nv_bfloat16* X = (which ? p.pool_k : p.pool_q) + (size_t)bh * N * kD;
            int r = rb + lane;
            r += r < 0 ? g.H : 0;
            const uint32_t dst = smem_u32(buf) + lane * 8 * kD * 2;
            // columns cb .. cb + 7 with -W < cb <= W - 8, each negative one taken + W
            if (cb >= 0 || cb <= -8) {  // one run of 8 columns
                bulk_load(dst, X + (size_t)(r * g.W + (cb < 0 ? cb + g.W : cb)) * kD, 8 * kD * 2, bar);
            } else {  // columns W + cb .. W - 1, then 0 .. 7 + cb
                const int n1 = -cb;  // 1 .. 7
                bulk_load(dst, X + (size_t)(r * g.W + g.W + cb) * kD, n1 * kD * 2, bar);
                bulk_load(dst + n1 * kD * 2, X + (size_t)r * g.W * kD, (8 - n1) * kD * 2, bar);
            }
        }
        if (!mbar_wait(bar, round & 1, abortf, p.budget_ns)) {
            volatile int never = 0;  // wait once more, for the copies only, before giving up
            mbar_wait(bar, round & 1, &never, p.budget_ns);
            return false;
        }
        if (gwarp == 0 && lane == 0 && round == 0) TL_CTA(tl::kPoolLanded);
        float acc[VE];
#pragma unroll
        for (int e = 0; e < VE; ++e) acc[e] = 0.f;
#pragma unroll
        for (int i = 0; i < LOADS; ++i) {
            const int pos = r0 + i * RPI;
            const uint4 v = *reinterpret_cast<const uint4*>(buf + (pos * kD + col * VE) * 2);
            const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float2 f = __bfloat1622float2(h2[e]);
                acc[2 * e] += f.x;
                acc[2 * e + 1] += f.y;
            }
        }
#pragma unroll
        for (int o = CPR; o < 32; o <<= 1)
#pragma unroll
            for (int e = 0; e < VE; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
        if (r0 == 0) {
            float* dst = const_cast<float*>(which ? p.sel_kb : p.sel_qb) + ((size_t)bh * Tb + label) * kD + col * VE;
            constexpr float kInv = 1.0f / 64.0f;
            reinterpret_cast<float4*>(dst)[0] = make_float4(acc[0] * kInv, acc[1] * kInv, acc[2] * kInv, acc[3] * kInv);
            reinterpret_cast<float4*>(dst)[1] = make_float4(acc[4] * kInv, acc[5] * kInv, acc[6] * kInv, acc[7] * kInv);
        }
    }
    return true;
}

// Grid-wide barrier for a persistent launch whose CTAs are all resident (one per SM, grid at
// most the SM count; the next grid is released only after it). Called by one thread of each
// CTA after a CTA barrier: a release add makes the CTA's writes (ordered before it by that
// barrier) visible with its arrival, and an acquire load sees every other CTA's. w[0] counts
// arrivals; the reset is left to grid_barrier_depart at the end of the kernel, off the
// critical path. Bounded; returns false on timeout or abort.
__device__ bool grid_barrier_arrive_wait(unsigned* w, unsigned n, volatile int* abortf, uint64_t budget_ns,
                                         bool arrive)
{
    if (arrive) asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(w) : "memory");
    const uint64_t t0 = globaltimer_ns();
    for (;;) {
        unsigned v;
        asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(w) : "memory");
        if (v == n) return true;
        if (*abortf || globaltimer_ns() - t0 > budget_ns) return false;
    }
}

// After the whole CTA is done (every CTA of the grid has passed the barrier by then): w[1]
// counts departures, and the last CTA to leave sets both words back to zero, so a call that
// completes leaves the workspace zero-filled. (A CTA that gave up at the barrier does not
// depart; the workspace is then zeroed again by the caller, as after any timeout.)
__device__ void grid_barrier_depart(unsigned* w, unsigned n)
{
    if (atomicAdd(&w[1], 1u) == n - 1) {
        atomicExch(&w[0], 0u);
        atomicExch(&w[1], 0u);
    }
}

// A list entry: written earlier in this launch under in-kernel selection (read through L2),
// else read-only input.
__device__ __forceinline__ int ld_list(const TcParams& p, const int32_t* a) { return p.sel_qb ? __ldcg(a) : __ldg(a); }

// Score row and Top-k gating of one item (one warp), with the arithmetic and the selection code
// of the mask kernels (S_j = q_b . k_b[j], four interleaved partial sums over d combined in a
// fixed order; the total order of sel::rank_select, walked by sel::ballot_select on keys held
// in registers), so the same means give the same lists. kbs: the head's k_b
// staged in shared memory, the 16-byte chunk c4 of row j at chunk c4 ^ (j & 15) (two lanes per
// bank at most when 32 lanes read one column); qs: the item's q_b row in shared memory. Not
// inlined, so that its registers do not weigh on the pipeline roles.
template <int kPer>
__device__ __noinline__ void select_item(const TcParams& p, int item, int lane, const float* kbs, const float* qs,
                                         uint32_t* S)
{
    const int Tb = p.g.Tb();
    const bool stamp = threadIdx.x == 0 && item == sel_first_item(p, blockIdx.x, gridDim.x * kSlots);
    if (stamp) TL_CTA(tl::kSelStart);
    const float4* q4 = reinterpret_cast<const float4*>(qs);
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
            for (int c4 = 0; c4 < kD / 4; ++c4) {
                const float4 qv = q4[c4];
                const float4 kv = *reinterpret_cast<const float4*>(row + 4 * (c4 ^ sw));
                a[0] = fmaf(qv.x, kv.x, a[0]);
                a[1] = fmaf(qv.y, kv.y, a[1]);
                a[2] = fmaf(qv.z, kv.z, a[2]);
                a[3] = fmaf(qv.w, kv.w, a[3]);
            }
            const float acc = (a[0] + a[1]) + (a[2] + a[3]);
            if (p.sel_scores) p.sel_scores[(size_t)item * Tb + j] = acc;
            key[m] = sel::order_key(acc);
        }
    }
    (void)S;
    if (stamp) TL_CTA(tl::kScoresDone);
    sel::ballot_select<kPer>(key, Tb, p.keep, lane, const_cast<int32_t*>(p.idx) + (size_t)item * p.keep);
    if (stamp) TL_CTA(tl::kWalkDone);
    if (lane == 0) p.sel_cnt[item] = p.keep;
    __syncwarp();
}

// Piece k of pipeline v (V pipelines) from the schedule in shared memory.
__device__ __forceinline__ Piece get_piece(const TcParams& p, const SlotSmem& sm, int k, int v, int V)
{
    Piece pc;
    if (k < sm.nA) {
        const int4 e = sm.pieceA[k];
        pc.item = e.x;
        pc.tb = e.y;
        pc.nb = e.z;
        pc.part = e.w;
    } else {
        const int r = k - sm.nA;
        pc.item = p.sel_qb ? sel_first_item(p, v, V) + r : sm.M + v + r * V;
        pc.tb = 0;
        pc.part = -1;
        pc.nb = p.units;
        if (p.idx && !p.sel_qb)
            pc.nb = p.ntxt + min(max(r < kCntCap ? sm.cnts[r] : __ldg(p.cnt + pc.item), 0), p.keep);
    }
    return pc;
}

// Fills the schedule of pipeline v (thread t of its nthr threads); see the work-schedule
// comment above.
__device__ void build_schedule(const TcParams& p, SlotSmem& sm, int v, int V, int t, int nthr)
{
    const int M = split_items(p, V);
    const int rest = p.num_items - M - v;
    const int nB = p.sel_qb ? sel_item_count(p, v, V) : (rest > 0 ? (rest + V - 1) / V : 0);
    if (p.idx && !p.sel_qb)
        for (int r = t; r < nB && r < kCntCap; r += nthr) sm.cnts[r] = __ldg(p.cnt + M + v + r * V);
    if (t != 0) return;
    int nA = 0;
    if (M > 0) {
        const int U = p.units;
        const long long u0 = (long long)M * U * v / V, u1 = (long long)M * U * (v + 1) / V;
        const long long cut = u1 / U * U;  // start of the item holding unit u1 - 1
        auto add = [&](long long a, long long b) {   // piece over units [a, b) of one item
            const int item = (int)(a / U);
            const int tb = (int)(a - (long long)item * U), te = (int)(b - (long long)item * U);
            const int n = p.ntxt + (p.idx ? min(max(__ldg(p.cnt + item), 0), p.keep) : p.keep);
            sm.pieceA[nA++] = make_int4(item, tb, max(0, min(te, n) - tb), tb > 0 ? 1 : (te < U ? 0 : -1));
        };
        long long uend = u1;
        if (u1 % U != 0 && cut > u0) {  // the cut last item goes first
            add(cut, u1);
            uend = cut;
        }
        for (long long u = u0; u < uend;) {
            const long long next = min((u / U + 1) * U, uend);
            add(u, next);
            u = next;
        }
    }
    sm.nA = nA;
    sm.nB = nB;
    sm.M = M;
}

__global__ void __maxnreg__(80) ssba_attn_tc_kernel(const __grid_constant__ TileMaps maps,
                                                                    const TcParams p)
{
    extern __shared__ uint8_t smem_raw[];
    SmemLayout& cs = *reinterpret_cast<SmemLayout*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                    ~static_cast<uintptr_t>(1023));
    const int gwarp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) TL_CTA(tl::kEntry);
    // the pipelines' variables are defined after the pooling below, so that they are not live
    // across its call (at 80 registers a thread, values live across a call are spilled)
    {
    const int slot = gwarp / kSlotWarps;
    SlotSmem& sm = cs.slot[slot];
    if (threadIdx.x % (kSlotWarps * 32) == 0) {
        if (slot == 0) cs.abort_flag = 0;
        for (int s = 0; s < kKStages; ++s) {
            mbar_init(smem_u32(&sm.k_full[s]), 1);
            mbar_init(smem_u32(&sm.k_empty[s]), 1);
        }
        for (int s = 0; s < kVStages; ++s) {
            mbar_init(smem_u32(&sm.v_full[s]), 1);
            mbar_init(smem_u32(&sm.v_empty[s]), 1);
        }
        for (int b = 0; b < kSBuf; ++b) {
            mbar_init(smem_u32(&sm.s_full[b]), 1);
            mbar_init(smem_u32(&sm.s_free[b]), 1);
            mbar_init(smem_u32(&sm.p_full[b]), 4);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&sm.q_full[b]), 1);
            mbar_init(smem_u32(&sm.q_empty[b]), 1);
            mbar_init(smem_u32(&sm.stats_full[b]), 4);
            mbar_init(smem_u32(&sm.stats_free[b]), 4);
        }
        mbar_init(smem_u32(&sm.o_full), 1);
        mbar_init(smem_u32(&sm.o_free), 4);
        mbar_init(smem_u32(&sm.drain[0]), 1);
        mbar_init(smem_u32(&sm.drain[1]), 1);
        if (p.pool_q)
            for (int w = slot * kSlotWarps; w < (slot + 1) * kSlotWarps; ++w) mbar_init(smem_u32(&cs.pool_bar[w]), 1);
        fence_mbar_init();
    }
    const Grid g = p.g;
    for (int l = threadIdx.x; l < g.Tb() && l < kWinCap; l += kThreads) cs.win[l] = window_entry(g, l);
    }
    // everything above reads no input; the lists, counts and tensors may come from the grid
    // launched just before this one (programmatic dependent launch)
    grid_dep_wait();
    if (threadIdx.x == 0) TL_CTA(tl::kDepWait);
    bool pool_fail = false;
    if (p.pool_q) {
        // the block means of the whole layer: every warp of the grid one (block, tensor) unit,
        // then a grid barrier; the next grid is released only after it, so that it cannot take
        // an SM that one of these CTAs still waits for
        __syncthreads();  // the pooling barriers are initialised
        pool_fail = !pool_phase(p, cs, gwarp, lane, &cs.abort_flag);
        pool_fail = __syncthreads_or(pool_fail);  // also orders this CTA's means before the arrival
        if (threadIdx.x == 0) TL_CTA(tl::kPooled);
        if (threadIdx.x == 0 && !pool_fail)
            pool_fail = !grid_barrier_arrive_wait(p.gsync, gridDim.x, &cs.abort_flag, p.budget_ns,
                                                  p.withhold != 2 || blockIdx.x != 0);
        // on a timeout the means of other CTAs may be missing: the status is set, and the raised
        // abort flag makes every role leave at its first wait that does not complete at once
        // (lists selected from stale means still hold labels in [0, Tb)). No early return and
        // no condition on the selection: either costs the pipeline roles registers (spills).
        pool_fail = __syncthreads_or(pool_fail);
        if (threadIdx.x == 0) TL_CTA(tl::kBarrier);
        if (pool_fail && threadIdx.x == 0) {
            atomicExch(p.status, SSBA_ERR_TIMEOUT);
            cs.abort_flag = 1;
        }
    }
    grid_dep_launch();
    const int slot = gwarp / kSlotWarps;   // which pipeline of this CTA
    const int warp = gwarp % kSlotWarps;   // role within the pipeline
    SlotSmem& sm = cs.slot[slot];
    volatile int* abortf = &cs.abort_flag;
    // pipeline `slot` of CTA b is pipeline b + slot * gridDim.x of 2 * gridDim.x: the items
    // left over after whole rounds go to the first pipelines, one per CTA, and the other
    // pipeline of such a CTA finishes first and leaves it the SM
    const int vcta = slot * gridDim.x + blockIdx.x;
    const int vgrid = gridDim.x * kSlots;
    const Grid g = p.g;
    const int Tb = g.Tb();
    const int N = g.H * g.W;
    if (p.sel_qb) {
        // the lists of this CTA's items (the contiguous ranges of its two pipelines): the k_b
        // of the heads they touch are staged by all threads in the stage buffers of both
        // pipelines (free until the producers start), one asynchronous round per batch of
        // heads; then one warp per item
        const int f0 = sel_first_item(p, blockIdx.x, vgrid), n0 = sel_item_count(p, blockIdx.x, vgrid);
        const int f1 = sel_first_item(p, blockIdx.x + gridDim.x, vgrid);
        const int n1 = sel_item_count(p, blockIdx.x + gridDim.x, vgrid);
        // heads of the two ranges: [h0a, h0b] and [h1a, h1b], staged in that order
        const int h0a = f0 / Tb, h0b = n0 ? (f0 + n0 - 1) / Tb : h0a - 1;
        const int h1a = f1 / Tb, h1b = n1 ? (f1 + n1 - 1) / Tb : h1a - 1;
        const int nh0 = max(0, h0b - h0a + 1), nh = nh0 + max(0, h1b - h1a + 1);
        auto head_of = [&](int hi) { return hi < nh0 ? h0a + hi : h1a + (hi - nh0); };
        // staging: pipeline 0's k, v, q buffers end with the scratch (per warp 128 key words and
        // a 64-float query row, then up to kSelQRows shared query rows); the rest of them and
        // pipeline 1's hold the heads
        constexpr uint32_t kRegion = (kKStages + kVStages + 2) * kTileBytes;  // k, v, q of one pipeline
        constexpr int kSelQRows = 48;
        constexpr int kWarpScratch = 128 + kD;  // words per warp: keys, then its own query row
        constexpr uint32_t kScratch = (kThreads / 32) * kWarpScratch * 4 + kSelQRows * kD * 4;
        const uint32_t hb = (uint32_t)Tb * kD * 4;
        const int cap0 = (int)((kRegion - kScratch) / hb), cap = cap0 + (int)(kRegion / hb);
        uint8_t* r0 = &cs.slot[0].k[0][0];
        uint32_t* keys = reinterpret_cast<uint32_t*>(r0 + kRegion - kScratch) + gwarp * kWarpScratch;
        float* qrows = reinterpret_cast<float*>(r0 + kRegion - kScratch + (kThreads / 32) * kWarpScratch * 4);
        auto staged = [&](int hi) {
            return reinterpret_cast<float*>(hi < cap0 ? r0 + hi * hb : &cs.slot[1].k[0][0] + (hi - cap0) * hb);
        };
        auto item_of = [&](int q) { return q < n0 ? f0 + q : f1 + (q - n0); };
        for (int base = 0; base < nh; base += cap) {
            const int m = min(cap, nh - base);
            // asynchronous 16-byte copies, all in flight at once: the heads' k_b (chunk c4 of row
            // j to chunk c4 ^ (j & 15)) and, in the first round, the items' q_b rows
            for (int e = threadIdx.x; e < m * Tb * (kD / 4); e += kThreads) {
                const int hi = e / (Tb * (kD / 4)), rem = e - hi * Tb * (kD / 4);
                const int j = rem / (kD / 4), c4 = rem - j * (kD / 4);
                const float* src = p.sel_kb + ((size_t)head_of(base + hi) * Tb + j) * kD + 4 * c4;
                const uint32_t dst = smem_u32(staged(hi) + j * kD + 4 * (c4 ^ (j & 15)));
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
            }
            if (base == 0)
                for (int e = threadIdx.x; e < min(n0 + n1, kSelQRows) * (kD / 4); e += kThreads) {
                    const int q = e / (kD / 4), c4 = e - q * (kD / 4);
                    const float* src = p.sel_qb + (size_t)item_of(q) * kD + 4 * c4;
                    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(qrows + q * kD + 4 * c4)),
                                 "l"(src) : "memory");
                }
            asm volatile("cp.async.wait_all;" ::: "memory");
            __syncthreads();
            if (threadIdx.x == 0 && base == 0) TL_CTA(tl::kStaged);
            // the items whose head is in this batch
            for (int q = gwarp; q < n0 + n1; q += kThreads / 32) {
                const int item = item_of(q);
                const int h = item / Tb;
                const int hi = (q < n0 ? h - h0a : nh0 + h - h1a) - base;
                if (hi < 0 || hi >= m) continue;
                const float* qs = qrows + q * kD;
                if (q >= kSelQRows) {  // rows past the staged ones: this warp's own copy
                    float* own = reinterpret_cast<float*>(keys) + 128;  // after its keys
                    if (lane < kD / 4)
                        reinterpret_cast<float4*>(own)[lane] =
                            __ldcg(reinterpret_cast<const float4*>(p.sel_qb + (size_t)item * kD) + lane);
                    __syncwarp();
                    qs = own;
                }
                if (Tb <= 32) select_item<1>(p, item, lane, staged(hi), qs, keys);
                else if (Tb <= 64) select_item<2>(p, item, lane, staged(hi), qs, keys);
                else if (Tb <= 128) select_item<4>(p, item, lane, staged(hi), qs, keys);
                else select_item<8>(p, item, lane, staged(hi), qs, keys);
            }
            __syncthreads();
        }
        if (threadIdx.x == 0) TL_CTA(tl::kSelected);
    }
    build_schedule(p, sm, vcta, vgrid, threadIdx.x % (kSlotWarps * 32), kSlotWarps * 32);
    if (gwarp == 0 && lane < 12) tma_prefetch_desc(lane < 4 ? &maps.q[lane] : (lane < 8 ? &maps.k[lane - 4] : &maps.v[lane - 8]));
    if (gwarp == 1) {
        tmem_alloc(smem_u32(&cs.tmem_base), kTmemCols);
        tmem_relinquish();
    }
    // the stage buffers held the pooled rows and the staged means (generic accesses); the
    // producers' tensor copies (async proxy) overwrite them next
    if (p.sel_qb) fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = cs.tmem_base + slot * kSlotCols;
    bool dead = false;
    if (threadIdx.x == 0) TL_CTA(tl::kPipesStart);
    if (threadIdx.x % (kSlotWarps * 32) == 0) TL_ITEM(slot, 0u, tl::kPipeClock0);

    if (warp == 0 || warp == 2) {
        // ------------------------------------------------------------ TMA producers
        // Warp 0 loads each item's Q tile and the K tiles of its key blocks into the K ring,
        // warp 2 the V tiles into the V ring; one elected lane each, blocking (suspending)
        // waits. A K slot frees when its QK is done and a V slot when its PV is done, so the
        // rings do not wait on each other, and the two issuing threads overlap their TMA
        // issue latency (about 140 cycles per box per thread).
        const bool is_k = warp == 0;
        uint32_t g = 0, nq = 0;
        const int npieces = sm.nA + sm.nB;
        for (int pi = 0; !dead && pi < npieces; ++pi, ++nq) {
            const Piece pc = get_piece(p, sm, pi, vcta, vgrid);
            const int bh = pc.item / Tb, label = pc.item - bh * Tb;
            const int nblk = pc.nb;
            // item blocks [tb, tb + nblk): text blocks first (positions < ntxt), then the
            // listed image blocks, list entry (position - ntxt)
            const int ti0 = max(pc.tb, p.ntxt);
            const int nimg = max(0, pc.tb + nblk - ti0);
            const int32_t* list = p.idx ? p.idx + (size_t)pc.item * p.keep + (ti0 - p.ntxt) : nullptr;
            // all lanes fetch the piece's labels in one round and stage their window entries;
            // lane 0 then issues the copies (measured: faster than prefetching the labels one
            // piece ahead with cp.async)
            uint32_t* lab = reinterpret_cast<uint32_t*>(sm.labels[is_k ? 0 : 1]);
            for (int t = lane; t < nimg && t < kLabelCap; t += 32) {
                const int j = list ? clamp_label(ld_list(p, list + t), Tb) : ti0 - p.ntxt + t;
                lab[t] = j < kWinCap ? cs.win[j] : window_entry(p.g, j);
            }
            if (kChecked && is_k && list) {
                // this piece's entries ascending and in range (the one before it too, for a second
                // part), and the item's count in [0, keep]
                bool bad = false;
                for (int t = lane; t < nimg; t += 32) {
                    const int raw = ld_list(p, list + t);
                    bad |= raw < 0 || raw >= Tb;
                    if (t > 0 || ti0 > p.ntxt) bad |= raw <= ld_list(p, list + t - 1);
                }
                if (lane == 0 && !p.sel_qb) {
                    const int c = __ldg(p.cnt + pc.item);
                    bad |= c < 0 || c > p.keep;
                }
                if (__any_sync(0xffffffffu, bad) && lane == 0) atomicExch(p.status, SSBA_ERR_CHECK);
            }
            __syncwarp();
            if (lane == 0) {
                if (is_k) {
                    const uint32_t qb = nq & 1;
                    if (!mbar_wait(smem_u32(&sm.q_empty[qb]), ((nq >> 1) & 1) ^ 1, abortf, p.budget_ns)) dead = true;
                    if (!dead) {
                        mbar_arrive_expect_tx(smem_u32(&sm.q_full[qb]), kTileBytes);
                        window_boxes_e(maps.q, smem_u32(&sm.q[qb][0]), smem_u32(&sm.q_full[qb]),
                                       label < kWinCap ? cs.win[label] : window_entry(p.g, label), bh);
                    }
                }
                const uint32_t nst = is_k ? kKStages : kVStages;
                // text blocks of the piece (positions below ntxt): rows [64 tt, 64 tt + 64) of
                // the text keys / values, zero past T_txt
                const int te_txt = min(pc.tb + nblk, p.ntxt);
                for (int tt = pc.tb; tt < te_txt && !dead; ++tt, ++g) {
                    const uint32_t slot = g % nst;
                    uint64_t* empty = is_k ? &sm.k_empty[slot] : &sm.v_empty[slot];
                    uint64_t* full = is_k ? &sm.k_full[slot] : &sm.v_full[slot];
                    if (!mbar_wait(smem_u32(empty), ((g / nst) & 1) ^ 1, abortf, p.budget_ns)) {
                        dead = true;
                        break;
                    }
                    mbar_arrive_expect_tx(smem_u32(full), kTileBytes);
                    tma_load_3d(smem_u32(is_k ? &sm.k[slot][0] : &sm.v[slot][0]), is_k ? &maps.kt : &maps.vt,
                                smem_u32(full), 0, tt * 64, bh);
                }
                // image blocks of the piece: list entries [ti0 - ntxt, ti0 - ntxt + nimg)
                const bool hold = p.withhold == 1 && is_k && vcta == 0;  // test hook: never lands
                const uint32_t empty0 = smem_u32(is_k ? &sm.k_empty[0] : &sm.v_empty[0]);
                const uint32_t full0 = smem_u32(is_k ? &sm.k_full[0] : &sm.v_full[0]);
                const uint32_t tile0 = smem_u32(is_k ? &sm.k[0][0] : &sm.v[0][0]);
                const CUtensorMap* m4 = is_k ? maps.k : maps.v;
                for (int t = 0; t < nimg && !dead; ++t, ++g) {
                    uint32_t e;
                    if (t < kLabelCap) {
                        e = lab[t];
                    } else {
                        const int j = list ? clamp_label(ld_list(p, list + t), Tb) : ti0 - p.ntxt + t;
                        e = j < kWinCap ? cs.win[j] : window_entry(p.g, j);
                    }
                    const uint32_t slot = g % nst;
                    if (!mbar_wait(empty0 + 8 * slot, ((g / nst) & 1) ^ 1, abortf, p.budget_ns)) {
                        dead = true;
                        break;
                    }
                    mbar_arrive_expect_tx(full0 + 8 * slot, kTileBytes);
                    if (hold && g == 0) continue;
                    window_boxes_e(m4, tile0 + slot * kTileBytes, full0 + 8 * slot, e, bh);
                    TL_TILE(gwarp / kSlotWarps, g, is_k ? tl::kKIssue : tl::kVIssue);
                }
            }
            dead = __shfl_sync(0xffffffffu, dead, 0);
            g = __shfl_sync(0xffffffffu, g, 0);
        }
        if (dead && lane == 0) {
            // drain: wait for the copies this thread issued that may still be in flight
            const uint32_t nst = is_k ? kKStages : kVStages;
            for (uint32_t x = g > nst ? g - nst : 0; x < g; ++x)
                wait_raw(smem_u32(is_k ? &sm.k_full[x % nst] : &sm.v_full[x % nst]), (x / nst) & 1, p.budget_ns);
            if (is_k)
                for (uint32_t n = nq > 1 ? nq - 1 : 0; n <= nq; ++n)
                    wait_raw(smem_u32(&sm.q_full[n & 1]), (n >> 1) & 1, p.budget_ns);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ QK issuer
        // S_t = Q K_t^T into S buffer t % 3, once PV_{t-3} has read P_{t-3} from it.
        // MMAs and commits are issued under an elect.sync taken at the issue site: the
        // compiler then keeps the descriptors on the uniform datapath (measured: 4 MMAs +
        // commit issue in about 280 cycles, against about 480 under a precomputed lane test).
        // elect.sync picks the same lane of a full warp every time, so a commit always
        // follows the MMAs of its own thread.
        const bool leader = elect_one_sync();
        uint32_t gblk = 0, nloc = 0;
        const uint32_t kbase = smem_u32(&sm.k[0][0]);
        const int npieces = sm.nA + sm.nB;
        for (int pi = 0; !dead && pi < npieces; ++pi, ++nloc) {
            const Piece pc = get_piece(p, sm, pi, vcta, vgrid);
            const int nblk = pc.nb;
            const uint32_t qb = nloc & 1;
            const uint32_t qaddr = smem_u32(&sm.q[qb][0]);
            if (!mbar_wait(smem_u32(&sm.q_full[qb]), (nloc >> 1) & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            if (nblk == 0 && elect_one_sync()) mma_commit(smem_u32(&sm.q_empty[qb]));
            for (int t = 0; t < nblk; ++t) {
                const uint32_t gb = gblk + t, slot = gb % kKStages, sb = gb % kSBuf;
                if (gb >= (uint32_t)kSBuf &&
                    !mbar_wait(smem_u32(&sm.s_free[sb]), ((gb / kSBuf) - 1) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                if (lane == 0) TL_TILE(gwarp / kSlotWarps, gb, tl::kSFree);
                if (!mbar_wait(smem_u32(&sm.k_full[slot]), (gb / kKStages) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                if (elect_one_sync()) {
                    const uint64_t adesc = sdesc_sw128(qaddr, 16, 1024);
                    const uint64_t bdesc = sdesc_sw128(kbase + slot * kTileBytes, 16, 1024);
                    const uint32_t d = tbase + kColS + sb * 64;
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_ss(d, adesc + (uint64_t)(k * 2), bdesc + (uint64_t)(k * 2), kIdescQK, k > 0 ? 1u : 0u);
                    mma_commit(smem_u32(&sm.s_full[sb]));
                    mma_commit(smem_u32(&sm.k_empty[slot]));
                    if (t == nblk - 1) mma_commit(smem_u32(&sm.q_empty[qb]));  // last read of this Q tile
                    TL_TILE(gwarp / kSlotWarps, gb, tl::kQKIssue);
                }
                __syncwarp();
            }
            gblk += nblk;
        }
        if (dead && leader) {
            mma_commit(smem_u32(&sm.drain[0]));
            wait_raw(smem_u32(&sm.drain[0]), 0, p.budget_ns);
        }
    } else if (warp == 3) {
        // ------------------------------------------------------------ PV issuer
        // O += P_t V_t once the softmax has written P_t to shared memory and V_t has landed;
        // PVs of a pipeline are issued by this one thread, so they accumulate into O in order.
        const bool leader = elect_one_sync();
        uint32_t gblk = 0, nloc = 0;
        const uint32_t vbase = smem_u32(&sm.v[0][0]);
        const int npieces = sm.nA + sm.nB;
        for (int pi = 0; !dead && pi < npieces; ++pi, ++nloc) {
            const Piece pc = get_piece(p, sm, pi, vcta, vgrid);
            const int nblk = pc.nb;
            for (int t = 0; t < nblk; ++t) {
                const uint32_t gb = gblk + t, pb = gb % kSBuf, slot = gb % kVStages;
                if (!mbar_wait(smem_u32(&sm.p_full[pb]), (gb / kSBuf) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                if (t == 0 && nloc > 0 &&
                    !mbar_wait(smem_u32(&sm.o_free), (nloc - 1) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                if (!mbar_wait(smem_u32(&sm.v_full[slot]), (gb / kVStages) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                if (lane == 0) TL_TILE(gwarp / kSlotWarps, gb, tl::kPVReady);
                tc_fence_after();
                if (elect_one_sync()) {
                    const uint64_t vdesc = sdesc_sw128(vbase + slot * kTileBytes, 8192, 1024);
                    const uint32_t pcol = tbase + kColS + pb * 64;
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_ts(tbase + kColO, pcol + k * 8, vdesc + (uint64_t)(k * 128), kIdescPV,
                               (t > 0 || k > 0) ? 1u : 0u);
                    mma_commit(smem_u32(&sm.v_empty[slot]));
                    mma_commit(smem_u32(&sm.s_free[pb]));
                    TL_TILE(gwarp / kSlotWarps, gb, tl::kPVIssue);
                }
                __syncwarp();
            }
            if (dead) break;
            // an empty item writes no O, but o_full must still not run two phases ahead
            if (nblk == 0 && nloc > 0 &&
                !mbar_wait(smem_u32(&sm.o_free), (nloc - 1) & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            if (elect_one_sync()) mma_commit(smem_u32(&sm.o_full));
            __syncwarp();
            gblk += nblk;
        }
        if (dead && leader) {
            mma_commit(smem_u32(&sm.drain[1]));
            wait_raw(smem_u32(&sm.drain[1]), 0, p.budget_ns);
        }
    } else if (warp >= 4 && warp < 8) {
        // ------------------------------------------------------------ softmax
        const int quad = gwarp & 3;  // TMEM lane quadrant of this warp
        const int half = lane >> 4;
        const int row = quad * 16 + (lane & 15);
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        const float c = p.scale_log2;
        uint32_t gblk = 0, nloc = 0;
        const int npieces = sm.nA + sm.nB;
        for (int pi = 0; !dead && pi < npieces; ++pi, ++nloc) {
            const Piece pc = get_piece(p, sm, pi, vcta, vgrid);
            const int nblk = pc.nb;
            float m_used = 0.f, l = 0.f;
            for (int t = 0; t < nblk; ++t) {
                const uint32_t gb = gblk + t, sb = gb % kSBuf;
                if (!mbar_wait(smem_u32(&sm.s_full[sb]), (gb / kSBuf) & 1, abortf, p.budget_ns)) {
                    dead = true;
                    break;
                }
                if (quad == 0 && lane == 0) TL_TILE(gwarp / kSlotWarps, gb, tl::kSmxStart);
                tc_fence_after();
                const uint32_t scol = tbase + lane_off + kColS + sb * 64;
                uint32_t sr[32];
                tmem_ld_16x32bx2_x16_off32(scol, *reinterpret_cast<uint32_t(*)[16]>(&sr[0]));
                tmem_ld_16x32bx2_x16_off32(scol + 16, *reinterpret_cast<uint32_t(*)[16]>(&sr[16]));
                tmem_wait_ld();
                if (quad == 0 && lane == 0) TL_TILE(gwarp / kSlotWarps, gb, tl::kSLoaded);
                {
                    // the last text block: its columns past T_txt are zero-filled keys, not keys
                    const int tt = pc.tb + t, valid = p.t_txt - tt * 64;
                    if (tt < p.ntxt && valid < 64)
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (half * 32 + i >= valid) sr[i] = __float_as_uint(-INFINITY);
                }
                float mx;
                {
                    float t8[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        t8[i] = fmaxf(fmaxf(__uint_as_float(sr[i]), __uint_as_float(sr[i + 8])),
                                      fmaxf(__uint_as_float(sr[i + 16]), __uint_as_float(sr[i + 24])));
#pragma unroll
                    for (int i = 0; i < 4; ++i) t8[i] = fmaxf(t8[i], t8[i + 4]);
                    mx = fmaxf(fmaxf(t8[0], t8[1]), fmaxf(t8[2], t8[3]));
                }
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
                const float mx2 = mx * c;
                // lazy rescale: the running max is raised only when it grows by more than
                // 2^kRescaleLog2; O is then rescaled below, after P_t is stored (so that O
                // and S are never held in registers at the same time)
                bool rescale = false;
                float alpha = 1.f;
                if (t == 0) {
                    m_used = mx2;
                } else {
                    const bool need = mx2 > m_used + kRescaleLog2;
                    rescale = __any_sync(0xffffffffu, need);
                    if (need) {
                        alpha = fast_exp2(m_used - mx2);
                        m_used = mx2;
                    }
                }
                if (quad == 0 && lane == 0) TL_TILE(gwarp / kSlotWarps, gb, tl::kMaxDone);
                // x = s * c - m and the row sums in packed fp32x2 arithmetic (two lanes per op)
                uint32_t pk[16];
                const float2 c2 = make_float2(c, c), nm2 = make_float2(-m_used, -m_used);
                float2 ls2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const float2 x = __ffma2_rn(make_float2(__uint_as_float(sr[2 * i]), __uint_as_float(sr[2 * i + 1])),
                                                c2, nm2);
                    const float2 pp = make_float2(fast_exp2(x.x), fast_exp2(x.y));
                    ls2[i & 1] = __fadd2_rn(ls2[i & 1], pp);
                    pk[i] = pack_bf16(pp.x, pp.y);
                }
                const float2 lsum = __fadd2_rn(ls2[0], ls2[1]);
                l = fmaf(l, alpha, lsum.x + lsum.y);
                if (quad == 0 && lane == 0) TL_TILE(gwarp / kSlotWarps, gb, tl::kSmxExp);
                // P_t (bf16 pairs) into the first half of S_t's buffer, which S_t no longer needs
                if (quad == 0 && lane == 0) TL_TILE(gwarp / kSlotWarps, gb, tl::kPFree);
                const uint32_t pb = sb;
                tmem_st_16x32bx2_x16_off16(tbase + lane_off + kColS + pb * 64, pk);
                if (rescale) {
                    // O must hold every earlier PV before it is rescaled; PV_t waits for p_full
                    const uint32_t qb = (gb - 1) % kSBuf;
                    if (!mbar_wait(smem_u32(&sm.s_free[qb]), ((gb - 1) / kSBuf) & 1, abortf, p.budget_ns)) {
                        dead = true;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t ocol = tbase + lane_off + kColO;
                    uint32_t o[16];
#pragma unroll
                    for (int h2 = 0; h2 < 2; ++h2) {
                        tmem_ld_16x32bx2_x16_off32(ocol + h2 * 16, o);
                        tmem_wait_ld();
#pragma unroll
                        for (int i = 0; i < 16; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                        tmem_st_16x32bx2_x16_off32(ocol + h2 * 16, o);
                    }
                }
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&sm.p_full[pb]));
                if (quad == 0 && lane == 0) TL_TILE(gwarp / kSlotWarps, gb, tl::kPStored);
            }
            if (dead) break;
            // hand the row statistics to the epilogue warps
            const float ltot = l + __shfl_xor_sync(0xffffffffu, l, 16);
            const uint32_t eb = nloc & 1;
            if (!mbar_wait(smem_u32(&sm.stats_free[eb]), ((nloc >> 1) & 1) ^ 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            if (half == 0) sm.stats[eb][row] = make_float2(m_used, ltot);
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&sm.stats_full[eb]));
            gblk += nblk;
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int quad = gwarp & 3;
        const int half = lane >> 4;
        const int row = quad * 16 + (lane & 15);
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        uint32_t nloc = 0;
        const int npieces = sm.nA + sm.nB;
        for (int pi = 0; !dead && pi < npieces; ++pi, ++nloc) {
            const Piece pc = get_piece(p, sm, pi, vcta, vgrid);
            const int bh = pc.item / Tb, label = pc.item - bh * Tb;
            const uint32_t eb = nloc & 1;
            if (quad == 0 && lane == 0) TL_ITEM(gwarp / kSlotWarps, nloc, tl::kEpiStart);
            if (!mbar_wait(smem_u32(&sm.o_full), nloc & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            if (quad == 0 && lane == 0) TL_ITEM(gwarp / kSlotWarps, nloc, tl::kEpiO);
            tc_fence_after();
            uint32_t o[32];
            tmem_ld_16x32bx2_x16_off32(tbase + lane_off + kColO, *reinterpret_cast<uint32_t(*)[16]>(&o[0]));
            tmem_ld_16x32bx2_x16_off32(tbase + lane_off + kColO + 16, *reinterpret_cast<uint32_t(*)[16]>(&o[16]));
            tmem_wait_ld();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&sm.o_free));
            if (!mbar_wait(smem_u32(&sm.stats_full[eb]), (nloc >> 1) & 1, abortf, p.budget_ns)) {
                dead = true;
                break;
            }
            float2 st = sm.stats[eb][row];
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&sm.stats_free[eb]));

            if (pc.part >= 0) {
                // a cut item: publish this part, and if the other part is already there,
                // merge (each warp owns 16 rows, so the hand-off is per warp)
                const int bidx = pc.part == 1 ? vcta : vcta + 1;
                const size_t mine = (size_t)bidx * 2 + pc.part, other = mine ^ 1;
                float4* wo = reinterpret_cast<float4*>(p.ws_o + (mine * kRows + row) * kD + half * 32);
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    wo[i] = make_float4(__uint_as_float(o[4 * i]), __uint_as_float(o[4 * i + 1]),
                                        __uint_as_float(o[4 * i + 2]), __uint_as_float(o[4 * i + 3]));
                if (half == 0) p.ws_st[mine * kRows + row] = st;
                __threadfence();
                __syncwarp();
                int arrived = 0;
                if (lane == 0) arrived = atomicAdd(p.ws_cnt + bidx * 4 + quad, 1);
                arrived = __shfl_sync(0xffffffffu, arrived, 0);
                if (arrived == 0) continue;  // first here: the other part merges
                if (lane == 0) atomicExch(p.ws_cnt + bidx * 4 + quad, 0);  // ready for the next launch
                __threadfence();
                const float2 os = __ldcg(p.ws_st + other * kRows + row);
                const float4* oo = reinterpret_cast<const float4*>(p.ws_o + (other * kRows + row) * kD + half * 32);
                // an empty part (sum 0) contributes nothing; its O was never written
                const bool a_ok = st.y > 0.f, b_ok = os.y > 0.f;
                const float m = a_ok ? (b_ok ? fmaxf(st.x, os.x) : st.x) : os.x;
                const float wa = a_ok ? fast_exp2(st.x - m) : 0.f, wb = b_ok ? fast_exp2(os.x - m) : 0.f;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const float4 x = __ldcg(oo + i);
                    const float xb[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float a = a_ok ? __uint_as_float(o[4 * i + e]) * wa : 0.f;
                        o[4 * i + e] = __float_as_uint(b_ok ? fmaf(xb[e], wb, a) : a);
                    }
                }
                st = make_float2(m, (a_ok ? st.y * wa : 0.f) + (b_ok ? os.y * wb : 0.f));
            }

            const bool ok = st.y > 0.f;
            const float inv = ok ? 1.f / st.y : 0.f;
            const int tok = g.token(label, tile_row_pos(g, label, row));
            uint4 v[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                float f[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) f[e] = ok ? __uint_as_float(o[8 * i + e]) * inv : 0.f;
                v[i].x = pack_bf16(f[0], f[1]);
                v[i].y = pack_bf16(f[2], f[3]);
                v[i].z = pack_bf16(f[4], f[5]);
                v[i].w = pack_bf16(f[6], f[7]);
            }
            // lanes l and l ^ 16 hold the two halves of one row (chunks 0-3 and 4-7): swap two
            // chunks so that every store instruction writes whole 32-byte sectors
            uint4 s0 = half ? v[0] : v[1], s1 = half ? v[2] : v[3], r0v, r1v;
            r0v.x = __shfl_xor_sync(0xffffffffu, s0.x, 16); r0v.y = __shfl_xor_sync(0xffffffffu, s0.y, 16);
            r0v.z = __shfl_xor_sync(0xffffffffu, s0.z, 16); r0v.w = __shfl_xor_sync(0xffffffffu, s0.w, 16);
            r1v.x = __shfl_xor_sync(0xffffffffu, s1.x, 16); r1v.y = __shfl_xor_sync(0xffffffffu, s1.y, 16);
            r1v.z = __shfl_xor_sync(0xffffffffu, s1.z, 16); r1v.w = __shfl_xor_sync(0xffffffffu, s1.w, 16);
            uint4* rowp = reinterpret_cast<uint4*>(p.O + ((size_t)bh * N + tok) * kD);
            // chunk written by this lane in instruction i: 2i + half
            rowp[0 + half] = half ? r0v : v[0];
            rowp[2 + half] = half ? r1v : v[2];
            rowp[4 + half] = half ? v[1] : r0v;
            rowp[6 + half] = half ? v[3] : r1v;
            if (half == 0)
                p.lse[(size_t)bh * N + tok] = ok ? (st.x * 0.69314718055994531f + logf(st.y)) : -INFINITY;
            if (quad == 0 && lane == 0) TL_ITEM(gwarp / kSlotWarps, nloc, tl::kEpiDone);
        }
    }

    if (dead) atomicExch(p.status, SSBA_ERR_TIMEOUT);
    if (threadIdx.x % (kSlotWarps * 32) == 0) TL_CTA(slot == 0 ? tl::kSlot0End : tl::kSlot1End);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (gwarp == 1) tmem_dealloc(cs.tmem_base, kTmemCols);
    if (p.pool_q && threadIdx.x == 0 && !cs.abort_flag) grid_barrier_depart(p.gsync, gridDim.x);
    if (threadIdx.x == 0) TL_CTA(tl::kEnd);
}

// [B*heads][T][d] bf16 as a 3-D map with 64-row boxes (128-byte swizzle); rows past T read
// as zeros.
bool encode_rows_map(CUtensorMap* m, const void* base, int BH, int T)
{
    EncodeTiledFn fn = tensor_map_encoder();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)T, (cuuint64_t)BH};
    cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)T * kD * 2};
    cuuint32_t box[3] = {kD, 64, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int num_sms() { return device_sm_count(); }
PerDeviceOnce g_attn_attr;  // the kernel's shared-memory attributes, set once per device

}  // namespace

// Split-merge workspace: counters, then row statistics, then O parts, for one boundary
// per pipeline of the largest grid this device runs (two per SM) plus one.
namespace {
size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }
int max_grid() { return num_sms(); }
size_t ws_boundaries() { return (size_t)kSlots * max_grid() + 1; }
size_t ws_cnt_bytes() { return align256(ws_boundaries() * 4 * sizeof(int)); }
size_t ws_st_bytes() { return align256(ws_boundaries() * 2 * kRows * sizeof(float2)); }
size_t ws_o_bytes() { return ws_boundaries() * 2 * kRows * kD * sizeof(float); }
}  // namespace

// ... then 256 bytes for the grid barrier words of the launch that pools.
size_t attn_tc_workspace_bytes() { return ws_cnt_bytes() + ws_st_bytes() + align256(ws_o_bytes()) + 256; }

int launch_attn_tc_bf16(const ssba_desc& d, const Grid& g, int keep, float scale, const void* Q, const void* K,
                        const void* V, const int32_t* idx, const int32_t* cnt, void* O, float* lse, void* ws,
                        size_t ws_bytes, cudaStream_t st, uint64_t budget_ns, int withhold, const void* Kt,
                        const void* Vt, int t_txt, const float* sel_qb, const float* sel_kb, float* sel_scores,
                        bool pool)
{
    if (pool && (!ws || !sel_qb || !sel_kb)) {
        set_error("ssba_forward_fused: needs a forward workspace and the block-mean buffers");
        return SSBA_ERR_WORKSPACE;
    }
    if (sel_qb && (g.Tb() > kWinCap || t_txt > 0 || !idx || !cnt)) {
        set_error("ssba_forward_select: needs Tb <= 256, no text segment and list outputs");
        return SSBA_ERR_UNSUPPORTED;
    }
    if (d.head_dim != kD || g.blk != 8 || (g.sr % 4) || (g.sc % 4)) {
        set_error("ssba_forward (bf16): needs head_dim=64, block=8 and shifts that are multiples of 4");
        return SSBA_ERR_UNSUPPORTED;
    }
    if (g.H >= 32768 || g.W >= 32768) {
        set_error("ssba_forward (bf16): H_tok and W_tok must be below 32768");
        return SSBA_ERR_UNSUPPORTED;
    }
    if (ws && ws_bytes < attn_tc_workspace_bytes()) {
        set_error("ssba_forward (bf16): workspace of %zu bytes, %zu needed", ws_bytes, attn_tc_workspace_bytes());
        return SSBA_ERR_WORKSPACE;
    }
    const int BH = d.B * d.heads;
    TileMaps maps;
    memset(&maps, 0, sizeof(maps));
    if (!encode_window_maps(maps.q, Q, BH, g.H, g.W) || !encode_window_maps(maps.k, K, BH, g.H, g.W) ||
        !encode_window_maps(maps.v, V, BH, g.H, g.W)) {
        set_error("ssba_forward (bf16): cuTensorMapEncodeTiled failed");
        return SSBA_ERR_CUDA;
    }
    if (t_txt > 0 && (!encode_rows_map(&maps.kt, Kt, BH, t_txt) || !encode_rows_map(&maps.vt, Vt, BH, t_txt))) {
        set_error("ssba_forward_joint: cuTensorMapEncodeTiled failed for the text keys/values");
        return SSBA_ERR_CUDA;
    }
    TcParams p;
    p.O = static_cast<__nv_bfloat16*>(O);
    p.lse = lse;
    p.idx = idx;
    p.cnt = cnt;
    p.g = g;
    p.keep = keep;
    p.t_txt = t_txt > 0 ? t_txt : 0;
    p.ntxt = (p.t_txt + 63) / 64;
    p.units = p.ntxt + keep;
    p.num_items = BH * g.Tb();
    p.scale_log2 = scale * 1.4426950408889634f;
    p.budget_ns = budget_ns;
    p.withhold = withhold;
    p.sel_qb = sel_qb;
    p.sel_kb = sel_kb;
    p.sel_cnt = const_cast<int32_t*>(cnt);
    p.sel_scores = sel_scores;
    p.pool_q = pool ? static_cast<const __nv_bfloat16*>(Q) : nullptr;
    p.pool_k = pool ? static_cast<const __nv_bfloat16*>(K) : nullptr;
    p.gsync = pool ? reinterpret_cast<unsigned*>(static_cast<char*>(ws) + ws_cnt_bytes() + ws_st_bytes() +
                                                 align256(ws_o_bytes()))
                   : nullptr;
    p.status = device_status_word();
    if (!p.status) {
        set_error("ssba_forward (bf16): could not resolve the device status word");
        return SSBA_ERR_CUDA;
    }
    const size_t smem = sizeof(SmemLayout) + 1024;
    g_attn_attr.run([smem] {
        cudaFuncSetAttribute(ssba_attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        cudaFuncSetAttribute(ssba_attn_tc_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
    });
    // One CTA fits an SM (shared memory), so each CTA runs kSlots pipelines; the persistent
    // grid has one CTA per SM (fewer for small problems).
    const int want = (p.num_items + kSlots - 1) / kSlots;
    const int grid = want < max_grid() ? want : max_grid();
    p.split = 0;
    p.ws_cnt = nullptr;
    p.ws_st = nullptr;
    p.ws_o = nullptr;
    if (ws) {
        char* w = static_cast<char*>(ws);
        p.ws_cnt = reinterpret_cast<int*>(w);
        p.ws_st = reinterpret_cast<float2*>(w + ws_cnt_bytes());
        p.ws_o = reinterpret_cast<float*>(w + ws_cnt_bytes() + ws_st_bytes());
        // Equal shares of blocks only pay when some pipeline would otherwise take one item
        // more than another, and when items are long: a merge costs a few global-memory
        // round trips (about 5 us under load, measured), which 11-block items do not
        // earn back but 64-block items (dense) do (179 vs 198 us at 1024 px, 24 heads).
        p.split = (!sel_qb && p.units >= kSplitMinKeep && p.num_items >= kSlots * grid &&
                   p.num_items % (kSlots * grid) != 0)
                      ? 1 : 0;
    }
    // programmatic dependent launch: the kernel may start (barriers, tensor memory, window
    // table) while the previous grid on the stream finishes; it waits for that grid before
    // reading any input
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, ssba_attn_tc_kernel, maps, p);
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("ssba_attn_tc_kernel launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

// Timeline of the last launch of the attention kernel on the current device (timeline build only).
int timeline_read(unsigned long long* cta, unsigned* tile, unsigned* item)
{
#ifdef SSBA_TIMELINE
    if (cudaMemcpyFromSymbol(cta, tl::cta_ev, sizeof(tl::cta_ev)) != cudaSuccess ||
        cudaMemcpyFromSymbol(tile, tl::tile_ev, sizeof(tl::tile_ev)) != cudaSuccess ||
        cudaMemcpyFromSymbol(item, tl::item_ev, sizeof(tl::item_ev)) != cudaSuccess) {
        set_error("ssba_timeline_read: copy from the device failed");
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
#else
    (void)cta;
    (void)tile;
    (void)item;
    set_error("ssba_timeline_read: this library was built without -DSSBA_TIMELINE");
    return SSBA_ERR_UNSUPPORTED;
#endif
}

// Dense attention: the 128-token-tile kernel (attn_dense.cu) when N is a multiple of 128, else
// this kernel with no list, every key block visited in label order with query tiles of one 8x8
// block each (unshifted grid).
int launch_dense_tc_bf16(const ssba_desc& d, float scale, const void* Q, const void* K, const void* V, void* O,
                         float* lse, void* ws, size_t ws_bytes, cudaStream_t st)
{
    if (ws && ws_bytes < attn_tc_workspace_bytes()) {  // the rules of ssba_forward, whichever kernel runs
        set_error("ssba_forward_dense: workspace of %zu bytes, %zu needed", ws_bytes, attn_tc_workspace_bytes());
        return SSBA_ERR_WORKSPACE;
    }
    const int rc = launch_dense_m128(d, scale, Q, K, V, O, lse, st);
    if (rc != SSBA_ERR_UNSUPPORTED) return rc;
    if (d.head_dim != kD || d.H_tok % 8 || d.W_tok % 8) {
        set_error("ssba_forward_dense: needs head_dim=64 and H_tok, W_tok multiples of 8");
        return SSBA_ERR_UNSUPPORTED;
    }
    Grid g;
    g.H = d.H_tok;
    g.W = d.W_tok;
    g.blk = 8;
    g.sr = 0;
    g.sc = 0;
    g.bw = d.W_tok / 8;
    return launch_attn_tc_bf16(d, g, g.Tb(), scale, Q, K, V, nullptr, nullptr, O, lse, ws, ws_bytes, st);
}

}  // namespace ssba
