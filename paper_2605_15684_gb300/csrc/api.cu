// api.cu -- the extern "C" boundary declared in include/ssba.h: argument
// validation on the host, workspace carving, and kernel launches on the caller's
// stream. Nothing here allocates device memory.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>

#include "bwd_tile.cuh"
#include "common.cuh"
#include "window.cuh"

namespace ssba {

__device__ int g_status = 0;

EncodeTiledFn tensor_map_encoder()
{
    static EncodeTiledFn fn = [] {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess) {
            cudaGetLastError();
            return static_cast<EncodeTiledFn>(nullptr);
        }
        return reinterpret_cast<EncodeTiledFn>(ptr);
    }();
    return fn;
}

bool encode_window_maps(CUtensorMap* m4, const void* base, int BH, int H, int W)
{
    EncodeTiledFn fn = tensor_map_encoder();
    if (!fn) return false;
    constexpr cuuint64_t d = 64;
    const cuuint32_t cols[4] = {8, 8, 4, 4}, rows[4] = {8, 4, 8, 4};
    for (int s = 0; s < 4; ++s) {
        cuuint64_t dims[4] = {d, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)BH};
        cuuint64_t strides[3] = {d * 2, (cuuint64_t)W * d * 2, (cuuint64_t)H * W * d * 2};
        cuuint32_t box[4] = {(cuuint32_t)d, cols[s], rows[s], 1};
        cuuint32_t es[4] = {1, 1, 1, 1};
        CUresult r = fn(&m4[s], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, es,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return false;
    }
    return true;
}

int current_device()
{
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return -1;
    }
    return dev;
}

int device_sm_count()
{
    static int cache[kMaxDevices] = {};
    static std::mutex m;
    const int dev = current_device();
    if (dev < 0 || dev >= kMaxDevices) return 1;
    std::lock_guard<std::mutex> lock(m);
    if (cache[dev] > 0) return cache[dev];
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
        cudaGetLastError();
        return 1;
    }
    cache[dev] = n;
    return n;
}

uintptr_t current_context_id()
{
    typedef int (*CtxGetCurrentFn)(void**);
    static CtxGetCurrentFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &ptr, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<CtxGetCurrentFn>(ptr);
    });
    void* ctx = nullptr;
    if (!fn || fn(&ctx) != 0) return 0;
    return reinterpret_cast<uintptr_t>(ctx);
}

void* device_symbol_address(const void* symbol, void* (&cache)[kMaxDevices], uintptr_t (&ctx)[kMaxDevices],
                            std::mutex& m)
{
    const int dev = current_device();
    if (dev < 0 || dev >= kMaxDevices) return nullptr;
    const uintptr_t c = current_context_id();
    std::lock_guard<std::mutex> lock(m);
    if (!cache[dev] || ctx[dev] != c) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, symbol) != cudaSuccess || !p) {
            cudaGetLastError();
            return nullptr;
        }
        cache[dev] = p;
        ctx[dev] = c;
    }
    return cache[dev];
}

int* device_status_word()
{
    static void* addr[kMaxDevices] = {};
    static uintptr_t ctx[kMaxDevices] = {};
    static std::mutex m;
    return static_cast<int*>(device_symbol_address(reinterpret_cast<const void*>(&g_status), addr, ctx, m));
}

namespace {
thread_local char t_err[512] = "";

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Shared validation of a descriptor; fills the grid geometry and the keep count.
int check_desc(const ssba_desc* d, const char* who, Grid* g, int* keep)
{
    if (!d) {
        set_error("%s: null descriptor", who);
        return SSBA_ERR_INVALID;
    }
    if (d->B <= 0 || d->heads <= 0 || d->H_tok <= 0 || d->W_tok <= 0 || d->head_dim <= 0 || d->block <= 0) {
        set_error("%s: sizes must be positive (B=%d heads=%d H=%d W=%d d=%d block=%d)", who, d->B, d->heads,
                  d->H_tok, d->W_tok, d->head_dim, d->block);
        return SSBA_ERR_INVALID;
    }
    if (d->H_tok % d->block || d->W_tok % d->block) {
        set_error("%s: H_tok=%d and W_tok=%d must be multiples of block=%d", who, d->H_tok, d->W_tok, d->block);
        return SSBA_ERR_INVALID;
    }
    if (!(d->rho >= 0.0 && d->rho < 1.0)) {
        set_error("%s: rho=%g must satisfy 0 <= rho < 1", who, d->rho);
        return SSBA_ERR_INVALID;
    }
    if (d->dtype != SSBA_BF16 && d->dtype != SSBA_FP32) {
        set_error("%s: unknown dtype %d", who, d->dtype);
        return SSBA_ERR_INVALID;
    }
    if (!(d->softmax_scale >= 0.f) || std::isinf(d->softmax_scale)) {
        set_error("%s: softmax_scale must be finite and >= 0 (0 = 1/sqrt(head_dim))", who);
        return SSBA_ERR_INVALID;
    }
    const long long N = (long long)d->H_tok * d->W_tok;
    const long long total = N * d->B * d->heads * d->head_dim;
    if (total > (1LL << 40) || N > (1LL << 26)) {
        set_error("%s: tensor too large", who);
        return SSBA_ERR_INVALID;
    }
    g->H = d->H_tok;
    g->W = d->W_tok;
    g->blk = d->block;
    g->sr = ((d->shift_r % d->H_tok) + d->H_tok) % d->H_tok;
    g->sc = ((d->shift_c % d->W_tok) + d->W_tok) % d->W_tok;
    g->bw = d->W_tok / d->block;
    const int Tb = g->Tb();
    const int k_drop = (int)std::floor((double)Tb * d->rho);
    *keep = Tb - k_drop;
    if (*keep < 1) {
        set_error("%s: keep = Tb - floor(Tb*rho) = %d must be >= 1", who, *keep);
        return SSBA_ERR_INVALID;
    }
    return SSBA_OK;
}

float resolve_scale(const ssba_desc* d)
{
    return d->softmax_scale > 0.f ? d->softmax_scale : 1.0f / std::sqrt((float)d->head_dim);
}

size_t elem_size(const ssba_desc* d) { return d->dtype == SSBA_BF16 ? 2 : 4; }

}  // namespace

void set_error(const char* fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(t_err, sizeof(t_err), fmt, ap);
    va_end(ap);
}

}  // namespace ssba

using namespace ssba;

extern "C" {

int ssba_keep_count(const ssba_desc* desc)
{
    Grid g;
    int keep;
    if (check_desc(desc, "ssba_keep_count", &g, &keep) != SSBA_OK) return -1;
    return keep;
}

size_t ssba_mask_workspace_bytes(const ssba_desc* desc)
{
    Grid g;
    int keep;
    if (check_desc(desc, "ssba_mask_workspace_bytes", &g, &keep) != SSBA_OK) return 0;
    size_t one = (size_t)desc->B * desc->heads * g.Tb() * desc->head_dim * sizeof(float);
    one = (one + 255) & ~(size_t)255;
    return 2 * one;
}

int ssba_build_mask(const ssba_desc* desc, const void* Q, const void* K, int32_t* kv_idx, int32_t* kv_cnt,
                    float* scores_opt, void* workspace, size_t ws_bytes, void* stream)
{
    SSBA_NVTX_RANGE("ssba_build_mask");
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_build_mask", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!Q || !K || !kv_idx || !kv_cnt) {
        set_error("ssba_build_mask: Q, K, kv_idx and kv_cnt must be non-null");
        return SSBA_ERR_INVALID;
    }
    const size_t es = elem_size(desc);
    if ((desc->head_dim * es) % 16 || desc->head_dim > 256) {
        set_error("ssba_build_mask: head_dim*elem must be a multiple of 16 bytes and head_dim <= 256");
        return SSBA_ERR_UNSUPPORTED;
    }
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(kv_idx, 4) || !aligned(kv_cnt, 4) ||
        (scores_opt && !aligned(scores_opt, 4))) {
        set_error("ssba_build_mask: Q and K must be 16-byte aligned, outputs 4-byte aligned");
        return SSBA_ERR_INVALID;
    }
    const size_t need = ssba_mask_workspace_bytes(desc);
    if (!workspace || ws_bytes < need || !aligned(workspace, 16)) {
        set_error("ssba_build_mask: workspace of %zu bytes (16-byte aligned) required, got %zu", need, ws_bytes);
        return SSBA_ERR_WORKSPACE;
    }
    float* qb = static_cast<float*>(workspace);
    float* kb = reinterpret_cast<float*>(static_cast<char*>(workspace) + need / 2);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    rc = launch_mask_fused(*desc, g, keep, Q, K, kv_idx, kv_cnt, scores_opt, st);
    if (rc != SSBA_ERR_UNSUPPORTED) return rc;
    rc = launch_pool(*desc, g, Q, K, qb, kb, st);
    if (rc != SSBA_OK) return rc;
    return launch_select(*desc, g, keep, qb, kb, kv_idx, kv_cnt, scores_opt, st);
}

int ssba_qkv_rope_pool(const ssba_desc* desc, const void* X, const void* Wqkv, const float* bias, void* Q, void* K,
                       void* V, float* qb, float* kb, void* stream)
{
    SSBA_NVTX_RANGE("ssba_qkv_rope_pool");
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_qkv_rope_pool", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!X || !Wqkv || !Q || !K || !V || (!qb) != (!kb)) {
        set_error("ssba_qkv_rope_pool: X, Wqkv, Q, K, V must be non-null, and qb, kb both set or both NULL");
        return SSBA_ERR_INVALID;
    }
    if (!aligned(X, 16) || !aligned(Wqkv, 16) || !aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) ||
        (bias && !aligned(bias, 16)) || (qb && (!aligned(qb, 16) || !aligned(kb, 16)))) {
        set_error("ssba_qkv_rope_pool: every device pointer must be 16-byte aligned");
        return SSBA_ERR_INVALID;
    }
    return launch_qkv_rope_pool(*desc, g, X, Wqkv, bias, Q, K, V, qb, kb, static_cast<cudaStream_t>(stream));
}

int ssba_select_mask(const ssba_desc* desc, const float* qb, const float* kb, int32_t* kv_idx, int32_t* kv_cnt,
                     float* scores_opt, void* stream)
{
    SSBA_NVTX_RANGE("ssba_select_mask");
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_select_mask", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!qb || !kb || !kv_idx || !kv_cnt) {
        set_error("ssba_select_mask: qb, kb, kv_idx and kv_cnt must be non-null");
        return SSBA_ERR_INVALID;
    }
    if (desc->head_dim % 4 || desc->head_dim > 256) {
        set_error("ssba_select_mask: head_dim must be a multiple of 4 and at most 256");
        return SSBA_ERR_UNSUPPORTED;
    }
    if (!aligned(qb, 16) || !aligned(kb, 16) || !aligned(kv_idx, 4) || !aligned(kv_cnt, 4) ||
        (scores_opt && !aligned(scores_opt, 4))) {
        set_error("ssba_select_mask: qb and kb must be 16-byte aligned, outputs 4-byte aligned");
        return SSBA_ERR_INVALID;
    }
    return launch_select(*desc, g, keep, qb, kb, kv_idx, kv_cnt, scores_opt, static_cast<cudaStream_t>(stream));
}

size_t ssba_forward_workspace_bytes(const ssba_desc* desc)
{
    Grid g;
    int keep;
    if (check_desc(desc, "ssba_forward_workspace_bytes", &g, &keep) != SSBA_OK) return 0;
    if (desc->dtype != SSBA_BF16) return 0;
    return attn_tc_workspace_bytes();
}

int ssba_forward(const ssba_desc* desc, const void* Q, const void* K, const void* V, const int32_t* kv_idx,
                 const int32_t* kv_cnt, void* O, float* lse, void* workspace, size_t ws_bytes, void* stream)
{
    SSBA_NVTX_RANGE("ssba_forward");
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_forward", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!Q || !K || !V || !kv_idx || !kv_cnt || !O || !lse) {
        set_error("ssba_forward: every pointer must be non-null");
        return SSBA_ERR_INVALID;
    }
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(O, 16) || !aligned(lse, 4) ||
        !aligned(kv_idx, 4) || !aligned(kv_cnt, 4)) {
        set_error("ssba_forward: Q, K, V, O must be 16-byte aligned; lse, kv_idx, kv_cnt 4-byte aligned");
        return SSBA_ERR_INVALID;
    }
    if (workspace && !aligned(workspace, 16)) {
        set_error("ssba_forward: workspace must be 16-byte aligned");
        return SSBA_ERR_INVALID;
    }
    const float scale = resolve_scale(desc);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (desc->dtype == SSBA_FP32)
        return launch_attn_simt_f32(*desc, g, keep, scale, static_cast<const float*>(Q),
                                    static_cast<const float*>(K), static_cast<const float*>(V), kv_idx, kv_cnt,
                                    static_cast<float*>(O), lse, st);
    return launch_attn_tc_bf16(*desc, g, keep, scale, Q, K, V, kv_idx, kv_cnt, O, lse, workspace, ws_bytes, st);
}

int ssba_pool_blocks(const ssba_desc* desc, const void* Q, const void* K, float* qb, float* kb, void* stream)
{
    SSBA_NVTX_RANGE("ssba_pool_blocks");
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_pool_blocks", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!Q || !K || !qb || !kb) {
        set_error("ssba_pool_blocks: Q, K, qb and kb must be non-null");
        return SSBA_ERR_INVALID;
    }
    if ((desc->head_dim * elem_size(desc)) % 16 || desc->head_dim > 256) {
        set_error("ssba_pool_blocks: head_dim*elem must be a multiple of 16 bytes and head_dim <= 256");
        return SSBA_ERR_UNSUPPORTED;
    }
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(qb, 16) || !aligned(kb, 16)) {
        set_error("ssba_pool_blocks: Q, K, qb and kb must be 16-byte aligned");
        return SSBA_ERR_INVALID;
    }
    return launch_pool_blocks(*desc, g, Q, K, qb, kb, static_cast<cudaStream_t>(stream));
}

namespace {
int forward_select_impl(const char* name, bool pool, const ssba_desc* desc, const void* Q, const void* K,
                        const void* V, const float* qb, const float* kb, int32_t* kv_idx, int32_t* kv_cnt,
                        float* scores_opt, void* O, float* lse, void* workspace, size_t ws_bytes, void* stream)
{
    Grid g;
    int keep;
    int rc = check_desc(desc, name, &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!Q || !K || !V || !qb || !kb || !kv_idx || !kv_cnt || !O || !lse) {
        set_error("%s: every pointer but scores_opt must be non-null", name);
        return SSBA_ERR_INVALID;
    }
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(O, 16) || !aligned(qb, 16) ||
        !aligned(kb, 16) || !aligned(lse, 4) || !aligned(kv_idx, 4) || !aligned(kv_cnt, 4) ||
        (scores_opt && !aligned(scores_opt, 4)) || (workspace && !aligned(workspace, 16))) {
        set_error("%s: Q, K, V, O, qb, kb, workspace 16-byte aligned; the rest 4-byte aligned", name);
        return SSBA_ERR_INVALID;
    }
    if (desc->dtype != SSBA_BF16) {
        set_error("%s: bf16 only (the tensor-core path)", name);
        return SSBA_ERR_UNSUPPORTED;
    }
    if (pool && !workspace) {
        set_error("%s: needs a workspace of ssba_forward_workspace_bytes(desc) bytes", name);
        return SSBA_ERR_WORKSPACE;
    }
    return launch_attn_tc_bf16(*desc, g, keep, resolve_scale(desc), Q, K, V, kv_idx, kv_cnt, O, lse, workspace,
                               ws_bytes, static_cast<cudaStream_t>(stream), kWaitBudgetNs, 0, nullptr, nullptr, 0, qb,
                               kb, scores_opt, pool);
}
}  // namespace

int ssba_forward_select(const ssba_desc* desc, const void* Q, const void* K, const void* V, const float* qb,
                        const float* kb, int32_t* kv_idx, int32_t* kv_cnt, float* scores_opt, void* O, float* lse,
                        void* workspace, size_t ws_bytes, void* stream)
{
    SSBA_NVTX_RANGE("ssba_forward_select");
    return forward_select_impl("ssba_forward_select", false, desc, Q, K, V, qb, kb, kv_idx, kv_cnt, scores_opt, O,
                               lse, workspace, ws_bytes, stream);
}

int ssba_forward_fused(const ssba_desc* desc, const void* Q, const void* K, const void* V, float* qb, float* kb,
                       int32_t* kv_idx, int32_t* kv_cnt, float* scores_opt, void* O, float* lse, void* workspace,
                       size_t ws_bytes, void* stream)
{
    SSBA_NVTX_RANGE("ssba_forward_fused");
    return forward_select_impl("ssba_forward_fused", true, desc, Q, K, V, qb, kb, kv_idx, kv_cnt, scores_opt, O, lse,
                               workspace, ws_bytes, stream);
}

int ssba_forward_joint(const ssba_desc* desc, const void* Q, const void* K, const void* V, const void* K_txt,
                       const void* V_txt, int32_t T_txt, const int32_t* kv_idx, const int32_t* kv_cnt, void* O,
                       float* lse, void* workspace, size_t ws_bytes, void* stream)
{
    SSBA_NVTX_RANGE("ssba_forward_joint");
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_forward_joint", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!Q || !K || !V || !kv_idx || !kv_cnt || !O || !lse || T_txt < 0 || (T_txt > 0 && (!K_txt || !V_txt))) {
        set_error("ssba_forward_joint: every pointer must be non-null (K_txt, V_txt when T_txt > 0) and T_txt >= 0");
        return SSBA_ERR_INVALID;
    }
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(O, 16) || !aligned(lse, 4) ||
        !aligned(kv_idx, 4) || !aligned(kv_cnt, 4) || (T_txt > 0 && (!aligned(K_txt, 16) || !aligned(V_txt, 16))) ||
        (workspace && !aligned(workspace, 16))) {
        set_error("ssba_forward_joint: Q, K, V, K_txt, V_txt, O and the workspace must be 16-byte aligned; lse, "
                  "kv_idx, kv_cnt 4-byte aligned");
        return SSBA_ERR_INVALID;
    }
    if (desc->dtype != SSBA_BF16) {
        set_error("ssba_forward_joint: bf16 only");
        return SSBA_ERR_UNSUPPORTED;
    }
    return launch_attn_tc_bf16(*desc, g, keep, resolve_scale(desc), Q, K, V, kv_idx, kv_cnt, O, lse, workspace,
                               ws_bytes, static_cast<cudaStream_t>(stream), kWaitBudgetNs, 0, K_txt, V_txt, T_txt);
}

int ssba_forward_dense(const ssba_desc* desc, const void* Q, const void* K, const void* V, void* O, float* lse,
                       void* workspace, size_t ws_bytes, void* stream)
{
    SSBA_NVTX_RANGE("ssba_forward_dense");
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_forward_dense", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!Q || !K || !V || !O || !lse) {
        set_error("ssba_forward_dense: every pointer must be non-null");
        return SSBA_ERR_INVALID;
    }
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(O, 16) || !aligned(lse, 4)) {
        set_error("ssba_forward_dense: Q, K, V, O must be 16-byte aligned; lse 4-byte aligned");
        return SSBA_ERR_INVALID;
    }
    if (workspace && !aligned(workspace, 16)) {
        set_error("ssba_forward_dense: workspace must be 16-byte aligned");
        return SSBA_ERR_INVALID;
    }
    if (desc->dtype != SSBA_BF16) {
        set_error("ssba_forward_dense: bf16 only");
        return SSBA_ERR_UNSUPPORTED;
    }
    return launch_dense_tc_bf16(*desc, resolve_scale(desc), Q, K, V, O, lse, workspace, ws_bytes,
                                static_cast<cudaStream_t>(stream));
}

int ssba_test_forward_timeout(const ssba_desc* desc, const void* Q, const void* K, const void* V,
                              const int32_t* kv_idx, const int32_t* kv_cnt, void* O, float* lse, uint64_t budget_ns,
                              void* stream)
{
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_test_forward_timeout", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!Q || !K || !V || !kv_idx || !kv_cnt || !O || !lse) {
        set_error("ssba_test_forward_timeout: every pointer must be non-null");
        return SSBA_ERR_INVALID;
    }
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(O, 16) || !aligned(lse, 4) ||
        !aligned(kv_idx, 4) || !aligned(kv_cnt, 4)) {
        set_error("ssba_test_forward_timeout: Q, K, V, O must be 16-byte aligned; lse, kv_idx, kv_cnt 4-byte aligned");
        return SSBA_ERR_INVALID;
    }
    if (desc->dtype != SSBA_BF16) {
        set_error("ssba_test_forward_timeout: bf16 only");
        return SSBA_ERR_UNSUPPORTED;
    }
    const uint64_t b = budget_ns < 1000000ull ? 1000000ull : (budget_ns > kWaitBudgetNs ? kWaitBudgetNs : budget_ns);
    return launch_attn_tc_bf16(*desc, g, keep, resolve_scale(desc), Q, K, V, kv_idx, kv_cnt, O, lse, nullptr, 0,
                               static_cast<cudaStream_t>(stream), b, 1);
}

int ssba_test_fused_timeout(const ssba_desc* desc, const void* Q, const void* K, const void* V, float* qb, float* kb,
                            int32_t* kv_idx, int32_t* kv_cnt, void* O, float* lse, void* workspace, size_t ws_bytes,
                            uint64_t budget_ns, void* stream)
{
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_test_fused_timeout", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!Q || !K || !V || !qb || !kb || !kv_idx || !kv_cnt || !O || !lse || !workspace) {
        set_error("ssba_test_fused_timeout: every pointer must be non-null");
        return SSBA_ERR_INVALID;
    }
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(O, 16) || !aligned(qb, 16) ||
        !aligned(kb, 16) || !aligned(lse, 4) || !aligned(kv_idx, 4) || !aligned(kv_cnt, 4) || !aligned(workspace, 16)) {
        set_error("ssba_test_fused_timeout: Q, K, V, O, qb, kb, workspace 16-byte aligned; the rest 4-byte aligned");
        return SSBA_ERR_INVALID;
    }
    if (desc->dtype != SSBA_BF16) {
        set_error("ssba_test_fused_timeout: bf16 only");
        return SSBA_ERR_UNSUPPORTED;
    }
    const uint64_t b = budget_ns < 1000000ull ? 1000000ull : (budget_ns > kWaitBudgetNs ? kWaitBudgetNs : budget_ns);
    return launch_attn_tc_bf16(*desc, g, keep, resolve_scale(desc), Q, K, V, kv_idx, kv_cnt, O, lse, workspace,
                               ws_bytes, static_cast<cudaStream_t>(stream), b, 2, nullptr, nullptr, 0, qb, kb, nullptr,
                               true);
}

size_t ssba_backward_workspace_bytes(const ssba_desc* desc)
{
    Grid g;
    int keep;
    if (check_desc(desc, "ssba_backward_workspace_bytes", &g, &keep) != SSBA_OK) return 0;
    return bwd::bwd_layout(*desc, g, keep).bytes;
}

int ssba_backward(const ssba_desc* desc, const void* Q, const void* K, const void* V, const void* O, const float* lse,
                  const void* dO, const int32_t* kv_idx, const int32_t* kv_cnt, float* dQ, float* dK, float* dV,
                  void* workspace, size_t ws_bytes, void* stream)
{
    SSBA_NVTX_RANGE("ssba_backward");
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_backward", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!Q || !K || !V || !O || !lse || !dO || !kv_idx || !kv_cnt || !dQ || !dK || !dV) {
        set_error("ssba_backward: every pointer must be non-null");
        return SSBA_ERR_INVALID;
    }
    // the kernels copy 16-byte chunks of the rows and store the gradients as float4
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(O, 16) || !aligned(dO, 16) ||
        !aligned(lse, 4) || !aligned(kv_idx, 4) || !aligned(kv_cnt, 4) || !aligned(dQ, 16) || !aligned(dK, 16) ||
        !aligned(dV, 16)) {
        set_error("ssba_backward: tensors must be 16-byte aligned; lse, kv_idx, kv_cnt 4-byte aligned");
        return SSBA_ERR_INVALID;
    }
    const size_t need = ssba_backward_workspace_bytes(desc);
    if (!workspace || ws_bytes < need || !aligned(workspace, 16)) {
        set_error("ssba_backward: workspace of %zu bytes (16-byte aligned) required, got %zu", need, ws_bytes);
        return SSBA_ERR_WORKSPACE;
    }
    return launch_backward(*desc, g, keep, resolve_scale(desc), Q, K, V, O, lse, dO, kv_idx, kv_cnt, dQ, dK, dV,
                           static_cast<float*>(workspace), static_cast<cudaStream_t>(stream));
}

int ssba_test_backward_timeout(const ssba_desc* desc, const void* Q, const void* K, const void* V, const void* O,
                               const float* lse, const void* dO, const int32_t* kv_idx, const int32_t* kv_cnt,
                               float* dQ, float* dK, float* dV, void* workspace, size_t ws_bytes, uint64_t budget_ns,
                               void* stream)
{
    Grid g;
    int keep;
    int rc = check_desc(desc, "ssba_test_backward_timeout", &g, &keep);
    if (rc != SSBA_OK) return rc;
    if (!Q || !K || !V || !O || !lse || !dO || !kv_idx || !kv_cnt || !dQ || !dK || !dV) {
        set_error("ssba_test_backward_timeout: every pointer must be non-null");
        return SSBA_ERR_INVALID;
    }
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(O, 16) || !aligned(dO, 16) ||
        !aligned(lse, 4) || !aligned(kv_idx, 4) || !aligned(kv_cnt, 4) || !aligned(dQ, 16) || !aligned(dK, 16) ||
        !aligned(dV, 16)) {
        set_error("ssba_test_backward_timeout: tensors 16-byte aligned; lse, kv_idx, kv_cnt 4-byte aligned");
        return SSBA_ERR_INVALID;
    }
    const size_t need = ssba_backward_workspace_bytes(desc);
    if (!workspace || ws_bytes < need || !aligned(workspace, 16)) {
        set_error("ssba_test_backward_timeout: workspace of %zu bytes (16-byte aligned) required, got %zu", need,
                  ws_bytes);
        return SSBA_ERR_WORKSPACE;
    }
    const uint64_t b = budget_ns < 1000000ull ? 1000000ull : (budget_ns > kWaitBudgetNs ? kWaitBudgetNs : budget_ns);
    rc = launch_backward_ws(*desc, g, keep, resolve_scale(desc), Q, K, V, O, lse, dO, kv_idx, kv_cnt, dQ, dK, dV,
                            workspace, static_cast<cudaStream_t>(stream), b, 1);
    if (rc == SSBA_ERR_UNSUPPORTED)
        set_error("ssba_test_backward_timeout: needs the persistent kernel (bf16, head_dim 64, shifts that are "
                  "multiples of 4, Tb <= 256)");
    return rc;
}

static int haar_args(const char* who, const void* in, const void* out, int N, int C, int H, int W, int nb,
                     int dtype)
{
    if (!in || !out || N <= 0 || C <= 0 || H <= 0 || W <= 0 || (H & 1) || (W & 1) || (nb != 3 && nb != 4) ||
        (dtype != SSBA_BF16 && dtype != SSBA_FP32)) {
        set_error("%s: needs non-null buffers, positive sizes, even H and W, nb 3 or 4 and a known dtype", who);
        return SSBA_ERR_INVALID;
    }
    if (!aligned(in, 16) || !aligned(out, 16)) {
        set_error("%s: buffers must be 16-byte aligned", who);
        return SSBA_ERR_INVALID;
    }
    return SSBA_OK;
}

int ssba_haar_dwt(const void* x, void* y, int32_t N, int32_t C, int32_t H, int32_t W, int32_t nb, int32_t dtype,
                  void* stream)
{
    SSBA_NVTX_RANGE("ssba_haar_dwt");
    int rc = haar_args("ssba_haar_dwt", x, y, N, C, H, W, nb, dtype);
    if (rc != SSBA_OK) return rc;
    return launch_haar(false, x, y, N, C, H, W, nb, dtype, static_cast<cudaStream_t>(stream));
}

int ssba_haar_iwt(const void* y, void* x, int32_t N, int32_t C, int32_t H, int32_t W, int32_t nb, int32_t dtype,
                  void* stream)
{
    SSBA_NVTX_RANGE("ssba_haar_iwt");
    int rc = haar_args("ssba_haar_iwt", y, x, N, C, H, W, nb, dtype);
    if (rc != SSBA_OK) return rc;
    return launch_haar(true, y, x, N, C, H, W, nb, dtype, static_cast<cudaStream_t>(stream));
}

static int pyramid_args(const char* who, const void* x, void* const* y, int N, int C, int H, int W, int levels,
                        int nb, int dtype)
{
    if (levels < 1 || levels > SSBA_HAAR_MAX_LEVELS || !y) {
        set_error("%s: levels must be 1..%d and y a host array of device pointers", who, SSBA_HAAR_MAX_LEVELS);
        return SSBA_ERR_INVALID;
    }
    const int m = 1 << levels;
    if (H <= 0 || W <= 0 || H % m || W % m) {
        set_error("%s: H and W must be positive multiples of 2^levels", who);
        return SSBA_ERR_INVALID;
    }
    for (int l = 0; l < levels; ++l) {
        int rc = haar_args(who, x, y[l], N, C, H >> l, W >> l, nb, dtype);
        if (rc != SSBA_OK) return rc;
    }
    return SSBA_OK;
}

int ssba_haar_dwt_pyramid(const void* x, void* const* y, int32_t N, int32_t C, int32_t H, int32_t W, int32_t levels,
                          int32_t nb, int32_t dtype, void* stream)
{
    SSBA_NVTX_RANGE("ssba_haar_dwt_pyramid");
    int rc = pyramid_args("ssba_haar_dwt_pyramid", x, y, N, C, H, W, levels, nb, dtype);
    if (rc != SSBA_OK) return rc;
    return launch_haar_pyramid(false, const_cast<void*>(x), y, N, C, H, W, levels, nb, dtype,
                               static_cast<cudaStream_t>(stream));
}

int ssba_haar_iwt_pyramid(void* const* y, void* x, int32_t N, int32_t C, int32_t H, int32_t W, int32_t levels,
                          int32_t nb, int32_t dtype, void* stream)
{
    SSBA_NVTX_RANGE("ssba_haar_iwt_pyramid");
    int rc = pyramid_args("ssba_haar_iwt_pyramid", x, y, N, C, H, W, levels, nb, dtype);
    if (rc != SSBA_OK) return rc;
    return launch_haar_pyramid(true, x, y, N, C, H, W, levels, nb, dtype, static_cast<cudaStream_t>(stream));
}

int ssba_get_status(int32_t* device_status_out)
{
    if (!device_status_out) {
        set_error("ssba_get_status: null output");
        return SSBA_ERR_INVALID;
    }
    int v = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_status, sizeof(int));
    if (e != cudaSuccess) {
        set_error("ssba_get_status: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    const int zero = 0;
    e = cudaMemcpyToSymbol(g_status, &zero, sizeof(int));
    if (e != cudaSuccess) {
        set_error("ssba_get_status: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    *device_status_out = v;
    return SSBA_OK;
}

const char* ssba_last_error(void) { return t_err; }

int ssba_timeline_read(uint64_t* cta, uint32_t* tile, uint32_t* item)
{
    if (!cta || !tile || !item) {
        set_error("ssba_timeline_read: null output");
        return SSBA_ERR_INVALID;
    }
    return timeline_read(reinterpret_cast<unsigned long long*>(cta), tile, item);
}

}  // extern "C"
