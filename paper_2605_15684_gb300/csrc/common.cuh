// common.cuh -- shared definitions of the CUDA library (not shared with the oracle).
#pragma once
#include <cstdint>
#include <mutex>
#include <utility>
#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include "ssba.h"

namespace ssba {

// NVTX ranges around the entry points that launch work (named after the entry point), so that a
// timeline profiler shows each call's host span beside its kernels; -DSSBA_NO_NVTX removes them.
// The markers cost a few nanoseconds when no profiler is attached.
#ifndef SSBA_NO_NVTX
#include <nvtx3/nvToolsExt.h>
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange&) = delete;
    NvtxRange& operator=(const NvtxRange&) = delete;
};
#define SSBA_NVTX_RANGE(name) ::ssba::NvtxRange ssba_nvtx_range_(name)
#else
#define SSBA_NVTX_RANGE(name) do { } while (0)
#endif

// Per-device host state. Devices are told apart by their ordinal (up to kMaxDevices); a launcher
// that caches something about a device (its SM count, a function attribute it has set, a
// symbol's address) keeps one entry per ordinal.
constexpr int kMaxDevices = 64;
// The current device's ordinal, or -1 if it cannot be read.
int current_device();
// SM count of the current device (1 when it cannot be read; not cached then).
int device_sm_count();
// The driver's cuTensorMapEncodeTiled, looked up once through the runtime (null if absent).
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn tensor_map_encoder();
// Opaque identity of the current context (0 if unknown): a cached device address is valid only
// in the context it was looked up in (cudaDeviceReset replaces the primary context).
uintptr_t current_context_id();
// Device address of a __device__ symbol on the current device, cached per device and context;
// nullptr on failure.
void* device_symbol_address(const void* symbol, void* (&cache)[kMaxDevices], uintptr_t (&ctx)[kMaxDevices],
                            std::mutex& m);

// Runs a function once per device (the current one), thread-safe: for settings such as
// cudaFuncSetAttribute that hold per device.
class PerDeviceOnce {
public:
    template <class F>
    void run(F&& f)
    {
        const int dev = current_device();
        if (dev < 0 || dev >= kMaxDevices) {
            f();
            return;
        }
        std::call_once(flags_[dev], std::forward<F>(f));
    }

private:
    std::once_flag flags_[kMaxDevices];
};

// Device address of the status word (SSBA_OK or SSBA_ERR_TIMEOUT) of the current
// device, read by ssba_get_status(); kernels that wait receive it as a parameter.
int* device_status_word();

// Token grid with the window shift of one layer (Sec. 2.2, Window Shift Strategy).
// A block label is row-major over the blk x blk tiles of the rolled grid; the
// token at in-block position (a, b) of label (br, bc) sits at rolled position
// (br*blk + a, bc*blk + b), i.e. at original position (rolled - shift) mod size.
struct Grid {
    int H, W, blk;
    int sr, sc;  // shifts reduced to [0, H) and [0, W)
    int bw;      // W / blk (labels per block-row)

    __host__ __device__ int Tb() const { return (H / blk) * bw; }

    __device__ __forceinline__ int token(int label, int pos) const
    {
        int br = label / bw, bc = label - br * bw;
        int a = pos / blk, b = pos - a * blk;
        int r = br * blk + a - sr;
        if (r < 0) r += H;
        int c = bc * blk + b - sc;
        if (c < 0) c += W;
        return r * W + c;
    }
};

// Host-side launchers (defined in the .cu files, called by api.cu).
int launch_pool(const ssba_desc& d, const Grid& g, const void* Q, const void* K, float* qb, float* kb,
                cudaStream_t st);
// Block means with the pooling arithmetic of the fused mask kernel (head_dim 64, 8x8 blocks;
// other shapes fall back to launch_pool), programmatic dependent launch.
int launch_pool_blocks(const ssba_desc& d, const Grid& g, const void* Q, const void* K, float* qb, float* kb,
                       cudaStream_t st);
int launch_select(const ssba_desc& d, const Grid& g, int keep, const float* qb, const float* kb,
                  int32_t* idx, int32_t* cnt, float* scores, cudaStream_t st);
// Pool + affinity + selection in one launch (head_dim 64, 8x8 blocks, Tb <= 256); returns
// SSBA_ERR_UNSUPPORTED without launching for other shapes.
int launch_mask_fused(const ssba_desc& d, const Grid& g, int keep, const void* Q, const void* K, int32_t* idx,
                      int32_t* cnt, float* scores, cudaStream_t st);
int launch_attn_simt_f32(const ssba_desc& d, const Grid& g, int keep, float scale, const float* Q,
                         const float* K, const float* V, const int32_t* idx, const int32_t* cnt, float* O,
                         float* lse, cudaStream_t st);
// budget_ns: wall-time limit of each barrier wait (a wait that runs out sets the device
// status to SSBA_ERR_TIMEOUT); withhold != 0 is the failure-detection test hook.
constexpr uint64_t kWaitBudgetNs = 2000000000ull;  // 2 s
int launch_attn_tc_bf16(const ssba_desc& d, const Grid& g, int keep, float scale, const void* Q,
                        const void* K, const void* V, const int32_t* idx, const int32_t* cnt, void* O,
                        float* lse, void* ws, size_t ws_bytes, cudaStream_t st,
                        uint64_t budget_ns = kWaitBudgetNs, int withhold = 0, const void* Kt = nullptr,
                        const void* Vt = nullptr, int t_txt = 0, const float* sel_qb = nullptr,
                        const float* sel_kb = nullptr, float* sel_scores = nullptr, bool pool = false);
// Dense attention with 128-token tiles (M=128 products; head_dim 64, bf16, N a multiple of 128);
// returns SSBA_ERR_UNSUPPORTED without launching for other shapes.
int launch_dense_m128(const ssba_desc& d, float scale, const void* Q, const void* K, const void* V, void* O,
                      float* lse, cudaStream_t st);
int launch_dense_tc_bf16(const ssba_desc& d, float scale, const void* Q, const void* K, const void* V,
                         void* O, float* lse, void* ws, size_t ws_bytes, cudaStream_t st);
// Bytes of the split-merge workspace of the bf16 forward on the current device.
size_t attn_tc_workspace_bytes();
// Copies out the attention kernel's time stamps (timeline build; else SSBA_ERR_UNSUPPORTED).
int timeline_read(unsigned long long* cta, unsigned* tile, unsigned* item);

int launch_backward(const ssba_desc& d, const Grid& g, int keep, float scale, const void* Q, const void* K,
                    const void* V, const void* O, const float* lse, const void* dO, const int32_t* idx,
                    const int32_t* cnt, float* dQ, float* dK, float* dV, float* Dbuf, cudaStream_t st);

// The same gradients on the tensor cores (bf16, head_dim 64, 8x8 blocks, Tb <= 256); returns
// SSBA_ERR_UNSUPPORTED without launching for other shapes.
int launch_backward_tc(const ssba_desc& d, const Grid& g, int keep, float scale, const void* Q, const void* K,
                       const void* V, const void* O, const float* lse, const void* dO, const int32_t* idx,
                       const int32_t* cnt, float* dQ, float* dK, float* dV, float* Dbuf, cudaStream_t st);
// The persistent warp-specialised tensor-core backward (bf16, head_dim 64, shifts that are
// multiples of 4, Tb <= 256); SSBA_ERR_UNSUPPORTED otherwise. workspace = the caller's
// ssba_backward workspace (bwd_layout).
int launch_backward_ws(const ssba_desc& d, const Grid& g, int keep, float scale, const void* Q, const void* K,
                       const void* V, const void* O, const float* lse, const void* dO, const int32_t* idx,
                       const int32_t* cnt, float* dQ, float* dK, float* dV, void* workspace, cudaStream_t st,
                       uint64_t budget_ns = kWaitBudgetNs, int withhold = 0);

int launch_haar(bool inverse, const void* in, void* out, int N, int C, int H, int W, int nb, int dtype,
                cudaStream_t st);
int launch_qkv_rope_pool(const ssba_desc& d, const Grid& g, const void* X, const void* Wqkv, const float* bias,
                         void* Q, void* K, void* V, float* qb, float* kb, cudaStream_t st,
                         uint64_t budget_ns = kWaitBudgetNs);

// Levels 1..SSBA_HAAR_MAX_LEVELS; ys holds one device pointer per level (host array).
int launch_haar_pyramid(bool inverse, void* x, void* const* ys, int N, int C, int H, int W, int L, int nb, int dtype,
                        cudaStream_t st);

// Thread-local error text for ssba_last_error().
void set_error(const char* fmt, ...);

}  // namespace ssba
