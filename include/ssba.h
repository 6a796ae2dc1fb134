/*
 * ssba.h -- C ABI of the GB300 (sm_103a) Shift Sparse Block Attention library.
 *
 * Shift Sparse Block Attention (SSBA) is defined in Sec. 2.2 of the ElasticDiT
 * paper: the image-token grid is cut into non-overlapping 8x8 token blocks (the
 * grid origin shifted by half a block on alternating layers, "Window Shift
 * Strategy"), each block's queries and keys are mean-pooled (Eq. for q_b, k_b),
 * the block affinity S = q_b k_b^T is formed, the k = floor(Tb * rho) smallest
 * entries of every row of S are masked ("Top-k Gating", Algorithm 1), and
 * softmax attention runs only over the key blocks that remain ("Efficient
 * Sparse Execution", Algorithm 1 SparseAttention).
 *
 * Conventions shared by every call
 *   Layout     Q, K, V, O are contiguous [B][heads][N][head_dim] with token
 *              n = r * W_tok + c on the row-major H_tok x W_tok grid.
 *   Ownership  The caller allocates every buffer (device memory unless a
 *              parameter says otherwise); the library allocates nothing and keeps
 *              no pointer after a call returns.
 *   Streams    `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *              stream). Every call only enqueues work and returns.
 *   Errors     Arguments are validated on the host; a bad descriptor, a null or
 *              misaligned pointer, or an unsupported shape returns a non-zero
 *              ssba_status and launches nothing. A failed launch returns
 *              SSBA_ERR_CUDA. A device-side failure (a bounded wait that ran out)
 *              is recorded in a device status word read by ssba_get_status().
 *              ssba_last_error() gives the thread's last message. Nothing aborts,
 *              throws across the ABI, or traps on the device.
 */
#ifndef SSBA_H_
#define SSBA_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SSBA_API __attribute__((visibility("default")))
#else
#define SSBA_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    SSBA_OK = 0,
    SSBA_ERR_INVALID = 1,     /* bad descriptor, null/misaligned pointer, bad sizes        */
    SSBA_ERR_UNSUPPORTED = 2, /* valid for the method but outside the kernels' fast path   */
    SSBA_ERR_CUDA = 3,        /* a CUDA runtime/driver call or launch failed               */
    SSBA_ERR_TIMEOUT = 4,     /* (device status) a bounded wait inside a kernel ran out    */
    SSBA_ERR_WORKSPACE = 5,   /* workspace missing or smaller than ssba_mask_workspace_bytes */
    SSBA_ERR_CHECK = 6        /* (device status, checked build only) an index list broke its
                                 invariants: a label outside [0, Tb), not ascending, or a
                                 count other than keep                                      */
} ssba_status;

typedef enum { SSBA_BF16 = 0, SSBA_FP32 = 1 } ssba_dtype;

/* One SSBA layer's geometry and sparsity rule.
 *   B, heads, head_dim   tensor sizes; head_dim = C of Sec. 2.2 (per head).
 *   H_tok, W_tok         image-token grid; both multiples of `block`.
 *   block                block side (8 in the paper: 8x8 = 64 tokens per block).
 *   shift_r, shift_c     window shift Delta of the layer (Sec. 2.2 Window Shift),
 *                        torch.roll semantics: token (r, c) moves to
 *                        ((r + shift_r) mod H_tok, (c + shift_c) mod W_tok) before
 *                        the unshifted partition. Any integer (reduced mod H, W).
 *   rho                  sparse ratio, 0 <= rho < 1; k_drop = floor(Tb * rho)
 *                        blocks are dropped per query block, keep = Tb - k_drop.
 *   dtype                ssba_dtype of Q, K, V and O.
 *   softmax_scale        scale of q.k inside the softmax; 0 selects 1/sqrt(head_dim). */
typedef struct {
    int32_t B, heads, H_tok, W_tok, head_dim;
    int32_t block;
    int32_t shift_r, shift_c;
    double rho;
    int32_t dtype;
    float softmax_scale;
} ssba_desc;

/* Number of key blocks kept per query block: Tb - floor(Tb * rho), Tb =
 * H_tok * W_tok / block^2 (Algorithm 1, "k <- floor(Tb * rho)" with k dropped).
 * Returns -1 for an invalid descriptor. */
SSBA_API int ssba_keep_count(const ssba_desc* desc);

/* Bytes of device workspace ssba_build_mask needs (the block means of Q and K
 * in fp32, 2 * B * heads * Tb * head_dim * 4 bytes, 256-byte aligned).
 * Returns 0 for an invalid descriptor. */
SSBA_API size_t ssba_mask_workspace_bytes(const ssba_desc* desc);

/* Builds the block mask of one layer (Sec. 2.2 Block Compression, Affinity
 * Matrix, Top-k Gating; Algorithm 1 partition .. Top-k Smallest).
 *   Q, K        device, [B][heads][N][head_dim] of desc->dtype (post-RoPE).
 *   kv_idx      device out, int32 [B][heads][Tb][keep]: for each query block, the
 *               labels of its kept key blocks in ascending order. Block label
 *               i = (u_r / block) * (W_tok / block) + (u_c / block) where
 *               (u_r, u_c) is the rolled position of the block's tokens.
 *   kv_cnt      device out, int32 [B][heads][Tb]: number of valid entries of
 *               each kv_idx row (always keep).
 *   scores_opt  device out or NULL, fp32 [B][heads][Tb][Tb]: the affinity S
 *               (block means, no scaling) the selection was made on.
 *   workspace   device scratch of at least ssba_mask_workspace_bytes(desc),
 *               16-byte aligned; contents are overwritten.
 * Ties in S keep the lower label. Any shift and head_dim in [1, 256] multiple of
 * 8 (bf16) or 4 (fp32) are supported. */
SSBA_API int ssba_build_mask(const ssba_desc* desc, const void* Q, const void* K, int32_t* kv_idx,
                    int32_t* kv_cnt, float* scores_opt, void* workspace, size_t ws_bytes,
                    void* stream);

/* Block-sparse attention forward (Sec. 2.2 Efficient Sparse Execution;
 * Algorithm 1 ExpandMask + SparseAttention, image tokens only): for every query
 * token n of block i = label(n), softmax over the keys of the blocks listed in
 * kv_idx[b][h][i][0 .. kv_cnt-1]:
 *   lse_n = ln sum_m exp(scale * q_n.k_m),  O_n = sum_m exp(scale * q_n.k_m - lse_n) v_m.
 *   Q, K, V     device, [B][heads][N][head_dim] of desc->dtype.
 *   kv_idx      device, int32 [B][heads][Tb][keep] labels in [0, Tb) (as written by
 *               ssba_build_mask for the same desc; any order, no repeats).
 *   kv_cnt      device, int32 [B][heads][Tb], each in [1, keep].
 *   O           device out, [B][heads][N][head_dim] of desc->dtype, original token order.
 *   lse         device out, fp32 [B][heads][N], natural log.
 *   workspace   device, optional (NULL and 0 allowed): the split-merge area of the
 *               bf16 kernel, at least ssba_forward_workspace_bytes(desc) bytes,
 *               16-byte aligned. With it, and with lists of at least 24 blocks, the
 *               persistent kernel gives its pipelines equal shares of key blocks and
 *               cuts at most one query block per share boundary in two, merging the
 *               parts' partial softmax sums; otherwise shares are whole query blocks
 *               (up to one query block's work of imbalance). The part that finishes
 *               second does the merge, so the rows of a cut query block may differ in
 *               their last bit from one call to the next (within the usual rounding).
 *               Rules: zero-fill it once before its first use. Every call that
 *               returns SSBA_OK and runs to completion leaves it zero-filled again,
 *               so later calls ordered after it on the GPU reuse it as is. Calls that
 *               may overlap on the GPU (two streams) need separate workspaces. After a
 *               call that ends with the device status SSBA_ERR_TIMEOUT, zero it again.
 *               fp32 ignores it.
 * bf16 runs on the tcgen05 tensor-core kernel and needs head_dim = 64, block = 8
 * and shifts that are multiples of 4; fp32 runs on the CUDA-core kernel with any
 * shift and head_dim = 64. Anything else returns SSBA_ERR_UNSUPPORTED. A workspace
 * smaller than required returns SSBA_ERR_WORKSPACE before any device work. */
SSBA_API int ssba_forward(const ssba_desc* desc, const void* Q, const void* K, const void* V,
                 const int32_t* kv_idx, const int32_t* kv_cnt, void* O, float* lse,
                 void* workspace, size_t ws_bytes, void* stream);

/* Joint text + image forward (Algorithm 1 with its text segment: the token mask is padded
 * with ones for the T_txt text tokens, Q, K and V are the concatenations [text; image], and
 * the image rows O[T_txt:] are returned). For every image query token n of block i:
 * softmax over all T_txt text keys and the image keys of the blocks listed in
 * kv_idx[b][h][i][0 .. kv_cnt-1]. Text queries are not evaluated, since Algorithm 1
 * returns the image features only.
 *   Q, K, V, kv_idx, kv_cnt, O, lse, workspace: as ssba_forward (image tokens only).
 *   K_txt, V_txt  device, [B][heads][T_txt][head_dim] bf16, 16-byte aligned.
 *   T_txt         number of text tokens, >= 0 (0 gives ssba_forward's result).
 * bf16 only, with the shape limits of the bf16 ssba_forward; text keys are read in
 * 64-token tiles, the last one masked past T_txt. */
SSBA_API int ssba_forward_joint(const ssba_desc* desc, const void* Q, const void* K, const void* V,
                                const void* K_txt, const void* V_txt, int32_t T_txt,
                                const int32_t* kv_idx, const int32_t* kv_cnt, void* O, float* lse,
                                void* workspace, size_t ws_bytes, void* stream);

/* Bytes of the optional ssba_forward / ssba_forward_dense / ssba_forward_select workspace, and
 * of the required one of ssba_forward_fused, for desc on the current device (it scales with the
 * device's SM count: about 10 MB on 152 SMs);
 * 0 for an fp32 or an invalid descriptor. Host only, no device work. */
SSBA_API size_t ssba_forward_workspace_bytes(const ssba_desc* desc);

/* Dense softmax attention over all N keys with the same layout and outputs as
 * ssba_forward (the 0% sparsity "baseline" of Table 2), from the same build:
 * bf16 only, head_dim = 64, H_tok and W_tok multiples of 8 (block is ignored).
 * Shift and rho are ignored. The workspace follows the rules of ssba_forward. */
SSBA_API int ssba_forward_dense(const ssba_desc* desc, const void* Q, const void* K, const void* V,
                       void* O, float* lse, void* workspace, size_t ws_bytes, void* stream);

/* Gradients of ssba_forward (the backward pass of Algorithm 1's SparseAttention over the
 * same kept blocks; the paper trains its sparse model but does not write the backward
 * out, so this is the chain rule of the forward). For the output gradient dO, with
 * p_nm = exp(scale q_n.k_m - lse_n) over the pairs the lists allow:
 *   D_n = dO_n . O_n,  dV_m = sum_n p_nm dO_n,  ds_nm = p_nm (dO_n . v_m - D_n),
 *   dQ_n = scale sum_m ds_nm k_m,  dK_m = scale sum_n ds_nm q_n.
 *   Q, K, V, O, dO  device, [B][heads][N][head_dim] of desc->dtype (O and lse as
 *                   ssba_forward wrote them), 16-byte aligned.
 *   lse             device, fp32 [B][heads][N], 4-byte aligned.
 *   kv_idx, kv_cnt  the lists of the forward, 4-byte aligned.
 *   dQ, dK, dV      device out, fp32 [B][heads][N][head_dim], 16-byte aligned, every element
 *                   written.
 *   workspace       device scratch of at least ssba_backward_workspace_bytes(desc) bytes
 *                   (the D_n values and the key blocks' transposed lists), 16-byte aligned,
 *                   one per stream (a call's kernels read what its own first kernel wrote).
 * bf16 inputs with head_dim = 64, 8x8 blocks and Tb <= 256 run on the tensor cores (tcgen05
 * products of 64-row tiles with fp32 accumulation in tensor memory; P and dS rounded to bf16
 * before their products, as the forward rounds P); fp32 inputs, and other shapes, on CUDA cores
 * in fp32. head_dim = 64 and block = 8 in both. Deterministic (no atomics: the key gradients are
 * gathered per key block over the query blocks that keep it). */
SSBA_API int ssba_backward(const ssba_desc* desc, const void* Q, const void* K, const void* V, const void* O,
                           const float* lse, const void* dO, const int32_t* kv_idx, const int32_t* kv_cnt,
                           float* dQ, float* dK, float* dV, void* workspace, size_t ws_bytes, void* stream);

/* Bytes of the ssba_backward workspace (0 for an invalid descriptor): D of every row
 * (B * heads * N * 4, rounded up to 256), then 256 bytes for a work counter, the transposed
 * lists (three int arrays of B * heads * Tb, B * heads * Tb and B * heads * Tb * keep entries)
 * and the rows' (lse, D) pairs by block (B * heads * N * 8 bytes), each part rounded up to 256
 * bytes. Every part is rewritten by each call: no zero-fill needed. */
SSBA_API size_t ssba_backward_workspace_bytes(const ssba_desc* desc);

/* Block compression alone (Sec. 2.2, the means q_b, k_b; Algorithm 1 MeanPool): the first
 * half of ssba_build_mask, for ssba_forward_select.
 *   Q, K    device, [B][heads][N][head_dim] of desc->dtype (post-RoPE), 16-byte aligned.
 *   qb, kb  device out, fp32 [B][heads][Tb][head_dim], 16-byte aligned.
 * Any shift; head_dim * element size a multiple of 16 bytes, head_dim <= 256. */
SSBA_API int ssba_pool_blocks(const ssba_desc* desc, const void* Q, const void* K, float* qb, float* kb,
                              void* stream);

/* Affinity, Top-k gating and sparse attention in one launch (Sec. 2.2, Algorithm 1 from
 * "S <- q_b k_b^T" on): each CTA computes the score rows and the kept-block lists of the query
 * blocks it will process (the arithmetic of ssba_build_mask, so the same means give the same
 * lists), writes them to kv_idx / kv_cnt (outputs here, same layout as ssba_build_mask), and
 * runs the forward of ssba_forward on them.
 *   qb, kb      device, fp32 block means from ssba_pool_blocks (or ssba_qkv_rope_pool).
 *   scores_opt  device out or NULL, fp32 [B][heads][Tb][Tb]: the scores of the selection.
 *   Q, K, V, O, lse, workspace as for ssba_forward.
 * bf16 only; Tb <= 256 (else SSBA_ERR_UNSUPPORTED: use ssba_build_mask + ssba_forward). */
SSBA_API int ssba_forward_select(const ssba_desc* desc, const void* Q, const void* K, const void* V,
                                 const float* qb, const float* kb, int32_t* kv_idx, int32_t* kv_cnt,
                                 float* scores_opt, void* O, float* lse, void* workspace, size_t ws_bytes,
                                 void* stream);

/* The whole of Algorithm 1 after RoPE in one launch (Sec. 2.2): block compression (the means
 * q_b, k_b, with the pooling arithmetic of ssba_pool_blocks, so the same Q, K give the same
 * means and lists), affinity, Top-k gating and the sparse attention. The persistent grid (one
 * CTA per SM) first pools every block of the layer into qb / kb, meets at a grid-wide barrier
 * (bounded wait; a timeout returns through ssba_get_status as SSBA_ERR_TIMEOUT, with O and
 * the lists not written), then runs ssba_forward_select on those means.
 *   qb, kb      device out, fp32 [B][heads][Tb][head_dim], 16-byte aligned: the block means.
 *   workspace   REQUIRED here, at least ssba_forward_workspace_bytes(desc) bytes: it holds the
 *               barrier's counters. The rules of ssba_forward's workspace hold (zero-filled before
 *               first use, left zero-filled, zeroed again after SSBA_ERR_TIMEOUT, one per stream).
 *   the rest    as ssba_forward_select.
 * The barrier needs every CTA of the grid (one per SM, at most the SM count) resident at once:
 * work on other streams that holds SMs for longer than the wait budget (2 s) makes the call end
 * with SSBA_ERR_TIMEOUT instead of waiting for it. The fallback with no grid-wide wait is
 * ssba_pool_blocks then ssba_forward_select on the same buffers (the same means, lists and
 * outputs); after SSBA_ERR_TIMEOUT, zero the workspace again before the next fused call.
 * bf16 only; Tb <= 256 (else SSBA_ERR_UNSUPPORTED); SSBA_ERR_WORKSPACE without a workspace. */
SSBA_API int ssba_forward_fused(const ssba_desc* desc, const void* Q, const void* K, const void* V, float* qb,
                                float* kb, int32_t* kv_idx, int32_t* kv_cnt, float* scores_opt, void* O,
                                float* lse, void* workspace, size_t ws_bytes, void* stream);

/* One level of the T-DVAE's 2-D Haar kernel bank F = {LL, HL, LH, HH} (Sec. 2.3
 * DWT-Enhanced Architecture), per channel, stride 2, orthonormal: for the window
 * a = x[2i][2j], b = x[2i][2j+1], c = x[2i+1][2j], d = x[2i+1][2j+1],
 *   LL = (a+b+c+d)/2, HL = (a-b+c-d)/2, LH = (a+b-c-d)/2, HH = (a-b-c+d)/2.
 *   x   device, [N][C][H][W] of dtype (SSBA_BF16 or SSBA_FP32), H and W even.
 *   y   device out, [N][nb*C][H/2][W/2] of dtype, subband-major (LL, HL, LH[, HH] of every
 *       channel); nb = 4, or 3 to keep c = {LL, HL, LH} as the paper's recursion does.
 * Both 16-byte aligned. fp32 arithmetic. Returns SSBA_ERR_INVALID for bad sizes or pointers,
 * SSBA_ERR_UNSUPPORTED when one image holds 2^31 or more 16-byte units (C*H*W*size >= 64 GiB). */
SSBA_API int ssba_haar_dwt(const void* x, void* y, int32_t N, int32_t C, int32_t H, int32_t W, int32_t nb,
                           int32_t dtype, void* stream);

/* The inverse level (the transpose of the orthonormal bank): y [N][nb*C][H/2][W/2] -> x
 * [N][C][H][W]; with nb = 3 the HH band is taken as zero. Same layouts and rules. */
SSBA_API int ssba_haar_iwt(const void* y, void* x, int32_t N, int32_t C, int32_t H, int32_t W, int32_t nb,
                           int32_t dtype, void* stream);

/* The encoder's Haar recursion (Sec. 2.3, the equation for W^(l)) without the stride-2
 * convolutions between levels, 1 <= levels <= SSBA_HAAR_MAX_LEVELS: level 1 is the bank on x,
 * level l the bank on the LL band of level l-1, all levels in one pass over x.
 *   x     device, [N][C][H][W] of dtype; H and W multiples of 2^levels.
 *   y     HOST array of `levels` device pointers; y[l-1] is [N][nb*C][H/2^l][W/2^l] of dtype,
 *         the layout of ssba_haar_dwt (nb = 3 leaves out HH; LL is always written).
 * All device buffers 16-byte aligned. Returns SSBA_ERR_INVALID for bad sizes or pointers. */
#define SSBA_HAAR_MAX_LEVELS 3
SSBA_API int ssba_haar_dwt_pyramid(const void* x, void* const* y, int32_t N, int32_t C, int32_t H, int32_t W,
                                   int32_t levels, int32_t nb, int32_t dtype, void* stream);

/* The decoder's inverse pyramid (Sec. 2.3) without the refinements between levels: the deepest
 * level's four bands (HH = 0 when nb = 3) and the detail bands HL, LH (, HH) of every shallower
 * level give x back; the LL bands of the shallower levels are not read. Same layouts. */
SSBA_API int ssba_haar_iwt_pyramid(void* const* y, void* x, int32_t N, int32_t C, int32_t H, int32_t W,
                                   int32_t levels, int32_t nb, int32_t dtype, void* stream);

/* The steps of Algorithm 1 before the mask, fused: the QKV projection of the image tokens,
 * RoPE on Q and K (Algorithm 1, first step; 2-D axial: dimensions [0, 32) turn with the
 * token's row, [32, 64) with its column, pair (2i, 2i+1) by pos * 10000^(-i/16)), and the
 * block compression of Sec. 2.2 (block means of Q and K over the layer's shifted 8x8 windows).
 *   X       device, bf16 [B][N][Dm], Dm = heads * 64, tokens in grid order (n = r * W_tok + c).
 *   Wqkv    device, bf16 [3 * Dm][Dm] (output channel-major: Q heads, then K, then V).
 *   bias    device fp32 [3 * Dm], or NULL.
 *   Q, K, V device out, bf16 [B][heads][N][64] (RoPE applied to Q and K).
 *   qb, kb  device out, fp32 [B][heads][Tb][64]: means of the bf16 Q and K over each block of
 *           the shifted grid (the layout ssba_select_mask reads); both NULL to skip them.
 * desc: dtype SSBA_BF16, head_dim 64, block 8, shifts multiples of 4. All device pointers
 * 16-byte aligned. fp32 accumulation. Returns SSBA_ERR_UNSUPPORTED for other shapes. */
SSBA_API int ssba_qkv_rope_pool(const ssba_desc* desc, const void* X, const void* Wqkv, const float* bias, void* Q,
                                void* K, void* V, float* qb, float* kb, void* stream);

/* The mask from block means already computed (Sec. 2.2 Affinity Matrix and Top-k Gating;
 * Algorithm 1 from "S <- q_b k_b^T" on): the second half of ssba_build_mask, for callers that
 * pooled in the projection (ssba_qkv_rope_pool).
 *   qb, kb  device, fp32 [B][heads][Tb][head_dim], 16-byte aligned.
 *   kv_idx, kv_cnt, scores_opt as for ssba_build_mask. Ties keep the lower label. */
SSBA_API int ssba_select_mask(const ssba_desc* desc, const float* qb, const float* kb, int32_t* kv_idx,
                              int32_t* kv_cnt, float* scores_opt, void* stream);

/* Size of the scratch area built into the library for ssba_build_mask_noalloc (4 MiB). */
#define SSBA_NOALLOC_SCRATCH_BYTES (4u << 20)

/* ssba_build_mask without a workspace argument: the same kernels and results as
 * ssba_build_mask, but the scratch (the pooled q_b and k_b) lives in a fixed
 * SSBA_NOALLOC_SCRATCH_BYTES area inside the library. The paper has no counterpart to this
 * call. It is for callers that cannot allocate device memory themselves, for example a
 * plug-in running inside a host runtime that owns all device memory and offers it no
 * workspace, or a latency-critical loop where a cudaMalloc/cudaFree pair (which can
 * synchronise the device) is not acceptable.
 *   Arguments, layouts and outputs are those of ssba_build_mask; the caller still passes
 *   Q, K and the output buffers.
 *   Size limit: a layer whose scratch (ssba_mask_workspace_bytes, 2 * B * heads * Tb *
 *   head_dim * 4 bytes in two 256-byte-aligned halves) exceeds SSBA_NOALLOC_SCRATCH_BYTES is
 *   rejected with SSBA_ERR_UNSUPPORTED and a message, before any device work. 1024 px and
 *   2048 px layers with B = 1 and 24 heads of 64 fit.
 *   Allocation: none. No cudaMalloc, cudaFree or allocating library routine is called; every
 *   GPU that loads the library holds the scratch area until the process exits.
 *   Set-up: the first call on each device looks up the area's device address with that
 *   device current (cudaGetSymbolAddress); make that first call before any stream capture.
 *   The address is kept per device and context: after a cudaDeviceReset the next call looks
 *   it up again (the area then starts afresh, which the build never relies on).
 *   Sharing: every call uses the same area, which keeps the last call's contents. Nothing in
 *   it needs to start at zero (the pooling kernel writes every value the selection kernel
 *   reads). Calls that overlap on the GPU -- on two streams, or from two host threads --
 *   race on the area and must be serialised by the caller. */
SSBA_API int ssba_build_mask_noalloc(const ssba_desc* desc, const void* Q, const void* K,
                                     int32_t* kv_idx, int32_t* kv_cnt, float* scores_opt,
                                     void* stream);

/* Test hook for failure detection (the paper has no counterpart): runs the bf16 forward
 * of ssba_forward with every barrier wait limited to budget_ns of wall time (clamped to
 * [1 ms, 2 s]) and one K tile copy of the first pipeline announced but never issued, so
 * that the waits on it run out. The kernel then stops all its roles, waits (bounded) for
 * its own copies and MMAs in flight, frees its tensor memory and returns; the device
 * status word reads SSBA_ERR_TIMEOUT (ssba_get_status, after a synchronize), O and lse
 * are undefined, and the context stays usable. No fault, trap or endless wait is
 * involved. Arguments as ssba_forward (workspace NULL); bf16 only. */
SSBA_API int ssba_test_forward_timeout(const ssba_desc* desc, const void* Q, const void* K, const void* V,
                                       const int32_t* kv_idx, const int32_t* kv_cnt, void* O, float* lse,
                                       uint64_t budget_ns, void* stream);

/* Test hook for failure detection in the fused launch (no counterpart in the paper): runs
 * ssba_forward_fused with every wait limited to budget_ns of wall time (clamped to [1 ms, 2 s])
 * and CTA 0 withholding its arrival at the grid barrier, so that every CTA's barrier wait runs
 * out. Each CTA then reports SSBA_ERR_TIMEOUT in the device status word, raises its abort flag
 * and leaves at its first wait that does not complete at once (the means are complete, so its
 * lists are valid); O, lse and the lists are undefined, the workspace's barrier words are left
 * set (zero it again, as after any timeout), and the context stays usable. No fault, trap or
 * endless wait is involved. Arguments as ssba_forward_fused (workspace required); bf16 only. */
SSBA_API int ssba_test_fused_timeout(const ssba_desc* desc, const void* Q, const void* K, const void* V, float* qb,
                                     float* kb, int32_t* kv_idx, int32_t* kv_cnt, void* O, float* lse,
                                     void* workspace, size_t ws_bytes, uint64_t budget_ns, void* stream);

/* Test hook for failure detection in the backward (no counterpart in the paper): runs the
 * persistent tensor-core kernel of ssba_backward with every wait limited to budget_ns of wall
 * time (clamped to [1 ms, 2 s]) and CTA 0 announcing its first pair's tile copies without
 * issuing them, so that the waits on them run out. That CTA stops all its roles, waits
 * (bounded) for its own copies and MMAs in flight, frees its tensor memory and returns; the
 * other CTAs finish their items. The device status word reads SSBA_ERR_TIMEOUT (ssba_get_status,
 * after a synchronize), dQ, dK and dV are undefined, and the context stays usable. No fault,
 * trap or endless wait is involved. Arguments as ssba_backward (workspace required); bf16,
 * head_dim 64, shifts that are multiples of 4 and Tb <= 256, else SSBA_ERR_UNSUPPORTED. */
SSBA_API int ssba_test_backward_timeout(const ssba_desc* desc, const void* Q, const void* K, const void* V,
                                        const void* O, const float* lse, const void* dO, const int32_t* kv_idx,
                                        const int32_t* kv_cnt, float* dQ, float* dK, float* dV, void* workspace,
                                        size_t ws_bytes, uint64_t budget_ns, void* stream);

/* Reads and clears the device status word of the current device (SSBA_OK or
 * SSBA_ERR_TIMEOUT). Synchronous: call after the caller's stream sync. Returns
 * SSBA_OK, or SSBA_ERR_CUDA if the read failed. */
SSBA_API int ssba_get_status(int32_t* device_status_out);

/* Message of the calling thread's last failed call ("" if none). */
SSBA_API const char* ssba_last_error(void);

/* Diagnostics (the paper has no counterpart): the time stamps that the attention kernel
 * (ssba_forward, ssba_forward_select, ssba_forward_fused, ...) recorded in its last launch on
 * the current device, in a library built with -DSSBA_TIMELINE (build.py variant "timeline").
 *   cta   host array of 256 x 16 uint64: per CTA, globaltimer nanoseconds of the launch's
 *         phases in this order: entry, dependency wait over, first pooled rows landed, means
 *         stored, grid barrier passed, head means staged, lists selected, pipelines start,
 *         pipeline 0 done, pipeline 1 done, exit, and for warp 0's first item the start of
 *         its selection, its score row done, its list done (0 where a phase did not run);
 *   tile  host array of 8 x 128 x 12 uint32: for pipelines 0 and 1 of CTAs 0, 1, grid/2 and
 *         grid-1, per tile (the pipeline's running key-block count), SM clock stamps of: K copy
 *         issued, QK issued, softmax saw S, softmax exps done, P stored, PV issued, V copy
 *         issued, QK's wait for a free S buffer over, S in the softmax's registers, row maxima
 *         known, P buffer free, PV's waits over;
 *   item  host array of 8 x 32 x 4 uint32: per item of those pipelines, SM clock stamps of: the
 *         epilogue starts waiting for O, O ready, the epilogue done, and (item 0 only) the
 *         pipeline's start.
 * Synchronous (call after the caller's stream sync). The default build records nothing and
 * returns SSBA_ERR_UNSUPPORTED; SSBA_ERR_CUDA if a copy fails. */
SSBA_API int ssba_timeline_read(uint64_t* cta, uint32_t* tile, uint32_t* item);

#ifdef __cplusplus
}
#endif

#endif /* SSBA_H_ */
