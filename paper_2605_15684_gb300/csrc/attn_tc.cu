// attn_tc.cu -- bf16 block-sparse attention forward on the sm_103a tensor cores
// (Sec. 2.2 "Efficient Sparse Execution": the kernel skips pruned blocks in its loads
// and its MMAs; Algorithm 1 SparseAttention over image tokens).
//
// Work item = one query block (64 tokens, an 8x8 window of the shifted grid) of one
// (batch, head); it visits only the key blocks listed for it. Per CTA (192 threads):
//   warp 0      TMA producer: for each listed key block, K and V land in a 5-stage
//               shared-memory ring as four 4x4-token boxes each (box = 64 d x 4 x 4 of a
//               [B*heads, H, W, d] tensor map, 128-byte swizzle). A half-block shift is a
//               multiple of 4 tokens, so every shifted 8x8 window is exactly four aligned
//               4x4 quadrants of the unshifted grid: no gather pass, no out-of-range fill.
//   warp 1      TMEM owner and MMA issuer (one elected lane):
//                 S_t = Q K_t^T   tcgen05.mma kind::f16, M=64 N=64, A = Q from TMEM,
//                                 B = K tile (K-major, SW128) from shared memory
//                 O  += P_t V_t   tcgen05.mma kind::f16, M=64 N=64, A = P from TMEM
//                                 (written over S_t), B = V tile (MN-major, SW128)
//               S is double-buffered so QK of block t+2 overlaps the softmax of t+1.
//   warps 2-5   softmax + epilogue, one TMEM lane quadrant each; the M=64 data path puts
//               query row r at lane 32*(r/16) + r%16, so two threads share a row (16x32bx2
//               TMEM loads), each holding 32 of its 64 scores. Online softmax in fp32 with
//               exp2 in the log2-scaled domain; the running max is only raised when it
//               grows by more than 2^8 (the O rescale then reads and writes O in TMEM),
//               which keeps P <= 256 in bf16 and l, O exact up to rounding.
//               They also stage the next item's Q into TMEM, and write O (bf16) and lse.
// All mbarrier waits are bounded (globaltimer budget + CTA abort flag); a timeout is
// reported in the device status word and the CTA drains its async work and exits.
#include <cuda.h>
#include <cstdio>

#include "common.cuh"
#include "ptx.cuh"

namespace ssba {

namespace {

using namespace ptx;

constexpr int kD = 64;
constexpr int kRows = 64;  // query rows per item = tokens per block
constexpr int kStages = 5;
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColS = 0;    // S/P double buffer: [0,64) and [64,128)
constexpr uint32_t kColO = 128;  // O accumulator: [128,192)
constexpr uint32_t kColQ = 192;  // Q double buffer: [192,224) and [224,256)
constexpr uint32_t kTileBytes = kRows * kD * 2;  // 8 KB
constexpr uint32_t kBoxBytes = 16 * kD * 2;      // 2 KB per 4x4 box
constexpr uint64_t kBudgetNs = 2000000000ull;    // 2 s per wait
constexpr float kRescaleLog2 = 8.0f;

// QK: M=64 N=64, A (Q) and B (K) K-major. PV: M=64 N=64, A (P) K-major, B (V) MN-major.
constexpr uint32_t kIdescQK = idesc_bf16_f32(64, 64, false, false);
constexpr uint32_t kIdescPV = idesc_bf16_f32(64, 64, false, true);

struct __align__(1024) SmemLayout {
    uint8_t k[kStages][kTileBytes];
    uint8_t v[kStages][kTileBytes];
    uint64_t kv_full[kStages];
    uint64_t kv_empty[kStages];
    uint64_t s_full[2];
    uint64_t p_full[2];
    uint64_t q_full[2];
    uint64_t pv_done;
    uint64_t o_full;
    uint64_t o_free;
    uint64_t drain;
    uint32_t tmem_base;
    int abort_flag;
};

struct TcParams {
    const __nv_bfloat16* Q;
    __nv_bfloat16* O;
    float* lse;
    const int32_t* idx;
    const int32_t* cnt;
    Grid g;
    int keep;
    int num_items;
    float scale_log2;  // softmax scale * log2(e)
    int* status;       // device status word
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

__device__ __forceinline__ bool wait_raw(uint32_t bar, uint32_t parity)
{
    uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity))
        if (globaltimer_ns() - t0 > kBudgetNs) return false;
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

// Key blocks of an item: the listed ones (count clamped to [0, keep]), or, in dense
// mode (no list), every block of the head.
__device__ __forceinline__ int item_nblk(const TcParams& p, int item)
{
    return p.idx ? min(max(__ldg(p.cnt + item), 0), p.keep) : p.keep;
}

__global__ void __launch_bounds__(kThreads, 2) ssba_attn_tc_kernel(const __grid_constant__ CUtensorMap tmK,
                                                                    const __grid_constant__ CUtensorMap tmV,
                                                                    const TcParams p)
{
    extern __shared__ uint8_t smem_raw[];
    SmemLayout& sm = *reinterpret_cast<SmemLayout*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                    ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abortf = &sm.abort_flag;
    const Grid g = p.g;
    const int Tb = g.Tb();
    const int N = g.H * g.W;

    if (threadIdx.x == 0) {
        sm.abort_flag = 0;
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&sm.kv_full[s]), 1);
            mbar_init(smem_u32(&sm.kv_empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&sm.s_full[b]), 1);
            mbar_init(smem_u32(&sm.p_full[b]), 4);
            mbar_init(smem_u32(&sm.q_full[b]), 4);
        }
        mbar_init(smem_u32(&sm.pv_done), 1);
        mbar_init(smem_u32(&sm.o_full), 1);
        mbar_init(smem_u32(&sm.o_free), 4);
        mbar_init(smem_u32(&sm.drain), 1);
        fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmK);
        tma_prefetch_desc(&tmV);
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
        const bool leader = elect_one_sync();
        uint32_t gkv = 0;
        for (int item = blockIdx.x; item < p.num_items && !dead; item += gridDim.x) {
            const int bh = item / Tb;
            const int nblk = item_nblk(p, item);
            const int32_t* list = p.idx ? p.idx + (size_t)item * p.keep : nullptr;
            for (int t = 0; t < nblk; ++t, ++gkv) {
                const uint32_t slot = gkv % kStages, ph = (gkv / kStages) & 1;
                if (!mbar_wait(smem_u32(&sm.kv_empty[slot]), ph ^ 1, abortf, kBudgetNs)) {
                    dead = true;
                    break;
                }
                if (leader) {
                    const int j = list ? clamp_label(__ldg(list + t), Tb) : t;
                    const int br = j / g.bw, bc = j - br * g.bw;
                    const uint32_t bar = smem_u32(&sm.kv_full[slot]);
                    mbar_arrive_expect_tx(bar, 2 * kTileBytes);
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        int r0 = br * 8 + (q >> 1) * 4 - g.sr;
                        if (r0 < 0) r0 += g.H;
                        int c0 = bc * 8 + (q & 1) * 4 - g.sc;
                        if (c0 < 0) c0 += g.W;
                        tma_load_4d(smem_u32(&sm.k[slot][q * kBoxBytes]), &tmK, bar, 0, c0, r0, bh);
                        tma_load_4d(smem_u32(&sm.v[slot][q * kBoxBytes]), &tmV, bar, 0, c0, r0, bh);
                    }
                }
                __syncwarp();
            }
        }
        if (dead && leader) {
            // drain: wait for the loads this warp issued that nobody consumed
            uint32_t first = gkv > (uint32_t)kStages ? gkv - kStages : 0;
            for (uint32_t x = first; x < gkv; ++x)
                wait_raw(smem_u32(&sm.kv_full[x % kStages]), (x / kStages) & 1);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        const bool leader = elect_one_sync();
        uint32_t gblk = 0, nloc = 0;
        const uint32_t kbase = smem_u32(&sm.k[0][0]);
        const uint32_t vbase = smem_u32(&sm.v[0][0]);
        for (int item = blockIdx.x; item < p.num_items && !dead; item += gridDim.x, ++nloc) {
            const int nblk = item_nblk(p, item);
            const uint32_t qcol = tbase + kColQ + (nloc & 1) * 32;
            if (!mbar_wait(smem_u32(&sm.q_full[nloc & 1]), (nloc >> 1) & 1, abortf, kBudgetNs)) {
                dead = true;
                break;
            }
            tc_fence_after();
            auto issue_qk = [&](uint32_t gb) -> bool {
                const uint32_t slot = gb % kStages;
                if (!mbar_wait(smem_u32(&sm.kv_full[slot]), (gb / kStages) & 1, abortf, kBudgetNs))
                    return false;
                tc_fence_after();
                if (leader) {
                    const uint64_t bdesc = sdesc_sw128(kbase + slot * kTileBytes, 16, 1024);
                    const uint32_t d = tbase + kColS + (gb & 1) * 64;
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_ts(d, qcol + k * 8, bdesc + (uint64_t)(k * 2), kIdescQK, k > 0 ? 1u : 0u);
                    mma_commit(smem_u32(&sm.s_full[gb & 1]));
                }
                __syncwarp();
                return true;
            };
            for (int t = 0; t < nblk && t < 2; ++t)
                if (!issue_qk(gblk + t)) {
                    dead = true;
                    break;
                }
            for (int t = 0; t < nblk && !dead; ++t) {
                const uint32_t gb = gblk + t, sb = gb & 1, slot = gb % kStages;
                if (!mbar_wait(smem_u32(&sm.p_full[sb]), (gb >> 1) & 1, abortf, kBudgetNs)) {
                    dead = true;
                    break;
                }
                if (t == 0 && nloc > 0 &&
                    !mbar_wait(smem_u32(&sm.o_free), (nloc - 1) & 1, abortf, kBudgetNs)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                if (leader) {
                    const uint64_t vdesc = sdesc_sw128(vbase + slot * kTileBytes, 8192, 1024);
                    const uint32_t pcol = tbase + kColS + sb * 64;
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_ts(tbase + kColO, pcol + k * 8, vdesc + (uint64_t)(k * 128), kIdescPV,
                               (t > 0 || k > 0) ? 1u : 0u);
                    mma_commit(smem_u32(&sm.kv_empty[slot]));
                    mma_commit(smem_u32(&sm.pv_done));
                }
                __syncwarp();
                if (t + 2 < nblk && !issue_qk(gb + 2)) {
                    dead = true;
                    break;
                }
            }
            if (dead) break;
            // an empty item writes no O, but o_full must still not run two phases ahead
            if (nblk == 0 && nloc > 0 &&
                !mbar_wait(smem_u32(&sm.o_free), (nloc - 1) & 1, abortf, kBudgetNs)) {
                dead = true;
                break;
            }
            if (leader) mma_commit(smem_u32(&sm.o_full));
            __syncwarp();
            gblk += nblk;
        }
        if (dead && leader) {
            mma_commit(smem_u32(&sm.drain));
            wait_raw(smem_u32(&sm.drain), 0);
        }
    } else {
        // ------------------------------------------------------------ softmax + epilogue
        const int quad = warp & 3;           // TMEM lane quadrant of this warp
        const int half = lane >> 4;          // which 32 of the row's 64 columns
        const int row = quad * 16 + (lane & 15);
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        const float c = p.scale_log2;
        uint32_t gblk = 0, nloc = 0;

        auto stage_q = [&](int item, uint32_t buf) {
            const int bh = item / Tb, label = item - (item / Tb) * Tb;
            const int tok = g.token(label, row);
            const uint4* src = reinterpret_cast<const uint4*>(p.Q + ((size_t)bh * N + tok) * kD + half * 32);
            uint32_t r[16];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                uint4 v = __ldg(src + i);
                r[4 * i] = v.x;
                r[4 * i + 1] = v.y;
                r[4 * i + 2] = v.z;
                r[4 * i + 3] = v.w;
            }
            tmem_st_16x32bx2_x16_off16(tbase + lane_off + kColQ + buf * 32, r);
            tmem_wait_st();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&sm.q_full[buf]));
        };

        if ((int)blockIdx.x < p.num_items) stage_q(blockIdx.x, 0);
        for (int item = blockIdx.x; item < p.num_items && !dead; item += gridDim.x, ++nloc) {
            const int bh = item / Tb, label = item - bh * Tb;
            const int nblk = item_nblk(p, item);
            if (item + (int)gridDim.x < p.num_items) stage_q(item + gridDim.x, (nloc + 1) & 1);

            float m_used = 0.f, l = 0.f;
            for (int t = 0; t < nblk; ++t) {
                const uint32_t gb = gblk + t, sb = gb & 1;
                if (!mbar_wait(smem_u32(&sm.s_full[sb]), (gb >> 1) & 1, abortf, kBudgetNs)) {
                    dead = true;
                    break;
                }
                tc_fence_after();
                const uint32_t scol = tbase + lane_off + kColS + sb * 64;
                uint32_t sr[32];
                tmem_ld_16x32bx2_x16_off32(scol, *reinterpret_cast<uint32_t(*)[16]>(&sr[0]));
                tmem_ld_16x32bx2_x16_off32(scol + 16, *reinterpret_cast<uint32_t(*)[16]>(&sr[16]));
                tmem_wait_ld();
                float mx = __uint_as_float(sr[0]);
#pragma unroll
                for (int i = 1; i < 32; ++i) mx = fmaxf(mx, __uint_as_float(sr[i]));
                mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
                const float mx2 = mx * c;
                if (t == 0) {
                    m_used = mx2;
                } else {
                    const bool need = mx2 > m_used + kRescaleLog2;
                    if (__any_sync(0xffffffffu, need)) {
                        // O must hold every earlier PV before it is rescaled
                        if (!mbar_wait(smem_u32(&sm.pv_done), (gb - 1) & 1, abortf, kBudgetNs)) {
                            dead = true;
                            break;
                        }
                        tc_fence_after();
                        const float alpha = need ? fast_exp2(m_used - mx2) : 1.f;
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
                        tmem_wait_st();
                        if (need) {
                            l *= alpha;
                            m_used = mx2;
                        }
                    }
                }
                uint32_t pk[16];
                float ls = 0.f;
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const float p0 = fast_exp2(fmaf(__uint_as_float(sr[2 * i]), c, -m_used));
                    const float p1 = fast_exp2(fmaf(__uint_as_float(sr[2 * i + 1]), c, -m_used));
                    ls += p0 + p1;
                    pk[i] = pack_bf16(p0, p1);
                }
                l += ls;
                tmem_st_16x32bx2_x16_off16(tbase + lane_off + kColS + sb * 64, pk);
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&sm.p_full[sb]));
            }
            if (dead) break;

            // ---- epilogue: O / l in bf16, lse = ln(sum exp(scale * s))
            const float ltot = l + __shfl_xor_sync(0xffffffffu, l, 16);
            if (!mbar_wait(smem_u32(&sm.o_full), nloc & 1, abortf, kBudgetNs)) {
                dead = true;
                break;
            }
            tc_fence_after();
            uint32_t o[32];
            tmem_ld_16x32bx2_x16_off32(tbase + lane_off + kColO, *reinterpret_cast<uint32_t(*)[16]>(&o[0]));
            tmem_ld_16x32bx2_x16_off32(tbase + lane_off + kColO + 16, *reinterpret_cast<uint32_t(*)[16]>(&o[16]));
            tmem_wait_ld();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&sm.o_free));

            const bool ok = ltot > 0.f;
            const float inv = ok ? 1.f / ltot : 0.f;
            const int tok = g.token(label, row);
            uint4* dst = reinterpret_cast<uint4*>(p.O + ((size_t)bh * N + tok) * kD + half * 32);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                uint4 v;
                v.x = pack_bf16(ok ? __uint_as_float(o[8 * i + 0]) * inv : 0.f, ok ? __uint_as_float(o[8 * i + 1]) * inv : 0.f);
                v.y = pack_bf16(ok ? __uint_as_float(o[8 * i + 2]) * inv : 0.f, ok ? __uint_as_float(o[8 * i + 3]) * inv : 0.f);
                v.z = pack_bf16(ok ? __uint_as_float(o[8 * i + 4]) * inv : 0.f, ok ? __uint_as_float(o[8 * i + 5]) * inv : 0.f);
                v.w = pack_bf16(ok ? __uint_as_float(o[8 * i + 6]) * inv : 0.f, ok ? __uint_as_float(o[8 * i + 7]) * inv : 0.f);
                dst[i] = v;
            }
            if (half == 0)
                p.lse[(size_t)bh * N + tok] = ok ? (m_used * 0.69314718055994531f + logf(ltot)) : -INFINITY;
            gblk += nblk;
        }
    }

    if (dead) atomicExch(p.status, SSBA_ERR_TIMEOUT);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tbase, kTmemCols);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn()
{
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    }
    return fn;
}

// [B*heads][H][W][d] bf16 viewed as a 4-D tensor map with a 64 x 4 x 4 x 1 box.
bool encode_qtile_map(CUtensorMap* m, const void* base, int BH, int H, int W)
{
    EncodeTiledFn fn = get_encode_fn();
    if (!fn) return false;
    cuuint64_t dims[4] = {(cuuint64_t)kD, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)BH};
    cuuint64_t strides[3] = {(cuuint64_t)kD * 2, (cuuint64_t)W * kD * 2, (cuuint64_t)H * W * kD * 2};
    cuuint32_t box[4] = {kD, 4, 4, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

int num_sms()
{
    static int n = 0;
    if (!n) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        if (n <= 0) n = 1;
    }
    return n;
}

}  // namespace

int launch_attn_tc_bf16(const ssba_desc& d, const Grid& g, int keep, float scale, const void* Q, const void* K,
                        const void* V, const int32_t* idx, const int32_t* cnt, void* O, float* lse,
                        cudaStream_t st)
{
    if (d.head_dim != kD || g.blk != 8 || (g.sr % 4) || (g.sc % 4)) {
        set_error("ssba_forward (bf16): needs head_dim=64, block=8 and shifts that are multiples of 4");
        return SSBA_ERR_UNSUPPORTED;
    }
    const int BH = d.B * d.heads;
    CUtensorMap tmK, tmV;
    if (!encode_qtile_map(&tmK, K, BH, g.H, g.W) || !encode_qtile_map(&tmV, V, BH, g.H, g.W)) {
        set_error("ssba_forward (bf16): cuTensorMapEncodeTiled failed");
        return SSBA_ERR_CUDA;
    }
    TcParams p;
    p.Q = static_cast<const __nv_bfloat16*>(Q);
    p.O = static_cast<__nv_bfloat16*>(O);
    p.lse = lse;
    p.idx = idx;
    p.cnt = cnt;
    p.g = g;
    p.keep = keep;
    p.num_items = BH * g.Tb();
    p.scale_log2 = scale * 1.4426950408889634f;
    p.status = device_status_word();
    if (!p.status) {
        set_error("ssba_forward (bf16): could not resolve the device status word");
        return SSBA_ERR_CUDA;
    }
    const size_t smem = sizeof(SmemLayout) + 1024;
    static bool attr_set = false;
    if (!attr_set) {
        cudaFuncSetAttribute(ssba_attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        attr_set = true;
    }
    const int grid = p.num_items < 2 * num_sms() ? p.num_items : 2 * num_sms();
    ssba_attn_tc_kernel<<<grid, kThreads, smem, st>>>(tmK, tmV, p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("ssba_attn_tc_kernel launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

// Dense attention from the same kernel: no list, every key block visited in label
// order with query tiles of one 8x8 block each (unshifted grid).
int launch_dense_tc_bf16(const ssba_desc& d, float scale, const void* Q, const void* K, const void* V, void* O,
                         float* lse, cudaStream_t st)
{
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
    return launch_attn_tc_bf16(d, g, g.Tb(), scale, Q, K, V, nullptr, nullptr, O, lse, st);
}

}  // namespace ssba
