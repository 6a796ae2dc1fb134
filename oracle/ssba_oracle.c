/*
 * ssba_oracle.c -- TEST INFRASTRUCTURE, not part of the product.
 *
 * A plain, slow, obviously-correct CPU statement in fp64 of Shift Sparse Block
 * Attention (SSBA) as the paper defines it (Sec. 2.2 "Sparse Block Attention",
 * Eq. for q_b/k_b, the affinity S = q_b k_b^T, Top-k gating, Algorithm 1, and the
 * "Window Shift Strategy" that follows it). Only the test-suite, the smoke check
 * and the CPU-baseline leg of the benchmark may load this library; the CUDA
 * library shares no code, header, table or helper with it.
 *
 * Every array is a single (batch, head) slice unless the name says "_all":
 *   X        [N][d]   image tokens, token n = r*W + c on an H x W grid (row-major)
 *   block_of [N]      block label of each token (Sec. 2.2 partition, shifted)
 *   Xb       [Tb][d]  block means
 *   S        [Tb][Tb] block affinity
 *   idx      [Tb][keep] kept key-block labels per query block, ascending
 *
 * Readings of the paper taken here (the paper is silent or ambiguous):
 *   - Top-k is taken per query-block row of S (k = floor(Tb*rho) counts a row).
 *   - k is the number of DROPPED blocks; keep = Tb - k.
 *   - Among equal S values, the higher key-block label is dropped first, so the
 *     lower label is kept.
 *   - The shift is a plain cyclic roll (torch.roll semantics): the rolled
 *     position of token (r, c) is ((r + s_r) mod H, (c + s_c) mod W) and blocks
 *     are the unshifted 8x8 tiles of the rolled grid.
 *   - Softmax scale is 1/sqrt(d) unless given; lse is a natural log of the sum of
 *     exp(scaled score).
 *   - Inputs are taken as post-RoPE (Algorithm 1 applies RoPE before pooling).
 *   - Text tokens (the _joint functions): the padded mask makes every text key visible to
 *     every image query; text queries are not evaluated, because Algorithm 1 returns
 *     the image rows O[T_txt:] only.
 *
 * Pins (tests/test_oracle_*.py): closed forms, brute force over block pairs,
 * brute-force subset search for the gate, np.roll for the partition, and the
 * rho = 0 reduction to dense softmax attention.
 */
#include <math.h>
#include <stdint.h>
#ifdef _OPENMP
#include <omp.h>
#endif
#include <stdlib.h>
#include <string.h>

#define ORC_OK 0
#define ORC_BAD 1

/* k = floor(Tb * rho) dropped blocks; keep = Tb - k (Sec. 2.2 Top-k gating,
 * Algorithm 1 "k <- floor(Tb * rho)"). */
int ssba_oracle_drop_count(int Tb, double rho)
{
    return (int)floor((double)Tb * rho);
}

int ssba_oracle_keep_count(int Tb, double rho)
{
    return Tb - ssba_oracle_drop_count(Tb, rho);
}

/* Partition into non-overlapping blk x blk blocks after shifting the grid
 * origin (Sec. 2.2 "Block Compression", Algorithm 1 partition step, and the
 * window-shift rule implemented with torch.roll).
 * torch.roll(x, shifts=s) moves the element at r to (r + s) mod H, so token
 * (r, c) sits at rolled position (u_r, u_c); the unshifted partition of the
 * rolled grid gives its block (u_r / blk, u_c / blk), labelled row-major. */
int ssba_oracle_partition(int H, int W, int blk, int shift_r, int shift_c,
                          int32_t *block_of)
{
    if (H <= 0 || W <= 0 || blk <= 0 || H % blk || W % blk || !block_of)
        return ORC_BAD;
    int sr = ((shift_r % H) + H) % H;
    int sc = ((shift_c % W) + W) % W;
    int bw = W / blk;
    for (int r = 0; r < H; ++r) {
        for (int c = 0; c < W; ++c) {
            int ur = (r + sr) % H;
            int uc = (c + sc) % W;
            block_of[r * W + c] = (ur / blk) * bw + (uc / blk);
        }
    }
    return ORC_OK;
}

/* Block compression: the mean of the tokens of each block (Eq. for
 * q_b = MeanPool(Q_img), k_b = MeanPool(K_img)). */
int ssba_oracle_pool(const double *X, int N, int d, const int32_t *block_of,
                     int Tb, double *Xb)
{
    if (!X || !block_of || !Xb || N <= 0 || d <= 0 || Tb <= 0) return ORC_BAD;
    int *count = (int *)calloc((size_t)Tb, sizeof(int));
    if (!count) return ORC_BAD;
    memset(Xb, 0, sizeof(double) * (size_t)Tb * d);
    for (int n = 0; n < N; ++n) {
        int b = block_of[n];
        if (b < 0 || b >= Tb) { free(count); return ORC_BAD; }
        count[b] += 1;
        for (int c = 0; c < d; ++c) Xb[(size_t)b * d + c] += X[(size_t)n * d + c];
    }
    for (int b = 0; b < Tb; ++b) {
        if (count[b] == 0) { free(count); return ORC_BAD; }
        for (int c = 0; c < d; ++c) Xb[(size_t)b * d + c] /= (double)count[b];
    }
    free(count);
    return ORC_OK;
}

/* Affinity matrix S = q_b k_b^T (Sec. 2.2 "Affinity Matrix"; no scaling). */
int ssba_oracle_affinity(const double *qb, const double *kb, int Tb, int d, double *S)
{
    if (!qb || !kb || !S || Tb <= 0 || d <= 0) return ORC_BAD;
    for (int i = 0; i < Tb; ++i) {
        for (int j = 0; j < Tb; ++j) {
            double acc = 0.0;
            for (int c = 0; c < d; ++c) acc += qb[(size_t)i * d + c] * kb[(size_t)j * d + c];
            S[(size_t)i * Tb + j] = acc;
        }
    }
    return ORC_OK;
}

/* Top-k gating (Sec. 2.2, Algorithm 1 "G <- Top-k Smallest(S, k)"): in each row,
 * the k_drop smallest entries of S are set to 0 in the gate G; the rest stay 1.
 * "Smallest" is the total order (S ascending, then label descending), so that of
 * two equal entries the higher label is dropped. The kept labels (G = 1) are
 * written in ascending order. */
int ssba_oracle_gate(const double *S, int Tb, int k_drop, int32_t *idx)
{
    if (!S || !idx || Tb <= 0 || k_drop < 0 || k_drop >= Tb) return ORC_BAD;
    unsigned char *G = (unsigned char *)malloc((size_t)Tb);
    if (!G) return ORC_BAD;
    int keep = Tb - k_drop;
    for (int i = 0; i < Tb; ++i) {
        const double *row = S + (size_t)i * Tb;
        for (int j = 0; j < Tb; ++j) G[j] = 1;
        for (int t = 0; t < k_drop; ++t) {
            int arg = -1;
            for (int j = 0; j < Tb; ++j) {
                if (!G[j]) continue;
                if (arg < 0 || row[j] < row[arg] || (row[j] == row[arg] && j > arg))
                    arg = j;
            }
            G[arg] = 0;
        }
        int w = 0;
        for (int j = 0; j < Tb; ++j)
            if (G[j]) idx[(size_t)i * keep + (w++)] = j;
        if (w != keep) { free(G); return ORC_BAD; }
    }
    free(G);
    return ORC_OK;
}

/* Tokens of every block in ascending token order: tok[start[b] .. start[b+1]). */
static int block_lists(int N, const int32_t *block_of, int Tb, int *start, int *tok)
{
    int *fill = (int *)calloc((size_t)Tb + 1, sizeof(int));
    if (!fill) return ORC_BAD;
    for (int b = 0; b <= Tb; ++b) start[b] = 0;
    for (int n = 0; n < N; ++n) {
        if (block_of[n] < 0 || block_of[n] >= Tb) { free(fill); return ORC_BAD; }
        start[block_of[n] + 1]++;
    }
    for (int b = 0; b < Tb; ++b) start[b + 1] += start[b];
    for (int n = 0; n < N; ++n) {
        int b = block_of[n];
        tok[start[b] + fill[b]++] = n;
    }
    free(fill);
    return ORC_OK;
}

/* One query row of the sparse attention (see ssba_oracle_attention). a and am are
 * scratch arrays of N entries. */
static int attend_row(const double *Q, const double *K, const double *V, int d, int n,
                      const int32_t *block_of, int Tb, const int32_t *idx, int keep,
                      double scale, const int *start, const int *tok, double *a, int *am,
                      double *O_row, double *lse_n)
{
    const int32_t *kept = idx + (size_t)block_of[n] * keep;
    int na = 0;
    for (int t = 0; t < keep; ++t) {
        int j = kept[t];
        if (j < 0 || j >= Tb) return ORC_BAD;
        for (int u = start[j]; u < start[j + 1]; ++u) {
            int m = tok[u];
            double dot = 0.0;
            for (int c = 0; c < d; ++c) dot += Q[(size_t)n * d + c] * K[(size_t)m * d + c];
            a[na] = scale * dot;
            am[na] = m;
            na++;
        }
    }
    double mx = -INFINITY;
    for (int u = 0; u < na; ++u) if (a[u] > mx) mx = a[u];
    double sum = 0.0;
    for (int u = 0; u < na; ++u) sum += exp(a[u] - mx);
    double l = mx + log(sum);
    *lse_n = l;
    for (int c = 0; c < d; ++c) O_row[c] = 0.0;
    for (int u = 0; u < na; ++u) {
        double p = exp(a[u] - l);
        const double *vm = V + (size_t)am[u] * d;
        for (int c = 0; c < d; ++c) O_row[c] += p * vm[c];
    }
    return ORC_OK;
}

/* Sparse attention restricted to the expanded mask (Sec. 2.2 "Efficient Sparse
 * Execution", Algorithm 1 ExpandMask + SparseAttention, image tokens only).
 * M(n, m) = 1 iff block_of[m] is among the kept labels of block_of[n]. For each
 * query n: a_m = scale * <Q_n, K_m> over the allowed keys, mx = max a_m,
 * lse_n = mx + ln sum exp(a_m - mx), O_n = sum exp(a_m - lse_n) V_m.
 * Keys are visited kept block by kept block in list order and, inside a block, in
 * ascending token order. Outputs are in the original token order. */
int ssba_oracle_attention(const double *Q, const double *K, const double *V,
                          int N, int d, const int32_t *block_of, int Tb,
                          const int32_t *idx, int keep, double scale,
                          double *O, double *lse)
{
    if (!Q || !K || !V || !block_of || !idx || !O || !lse) return ORC_BAD;
    if (N <= 0 || d <= 0 || Tb <= 0 || keep <= 0 || keep > Tb) return ORC_BAD;
    int *start = (int *)malloc(sizeof(int) * ((size_t)Tb + 1));
    int *tok = (int *)malloc(sizeof(int) * (size_t)N);
    double *a = (double *)malloc(sizeof(double) * (size_t)N);
    int *am = (int *)malloc(sizeof(int) * (size_t)N);
    int rc = (start && tok && a && am) ? block_lists(N, block_of, Tb, start, tok) : ORC_BAD;
    for (int n = 0; n < N && rc == ORC_OK; ++n)
        rc = attend_row(Q, K, V, d, n, block_of, Tb, idx, keep, scale, start, tok, a, am,
                        O + (size_t)n * d, lse + n);
    free(start); free(tok); free(a); free(am);
    return rc;
}

/* The same attention for the listed query tokens only: O_rows[r], lse_rows[r] are
 * the outputs of token rows[r]. Used to check full-size runs on sampled rows. */
int ssba_oracle_attention_rows(const double *Q, const double *K, const double *V,
                               int N, int d, const int32_t *block_of, int Tb,
                               const int32_t *idx, int keep, double scale,
                               const int32_t *rows, int nrows, double *O_rows, double *lse_rows)
{
    if (!Q || !K || !V || !block_of || !idx || !rows || !O_rows || !lse_rows) return ORC_BAD;
    if (N <= 0 || d <= 0 || Tb <= 0 || keep <= 0 || keep > Tb || nrows < 0) return ORC_BAD;
    int *start = (int *)malloc(sizeof(int) * ((size_t)Tb + 1));
    int *tok = (int *)malloc(sizeof(int) * (size_t)N);
    double *a = (double *)malloc(sizeof(double) * (size_t)N);
    int *am = (int *)malloc(sizeof(int) * (size_t)N);
    int rc = (start && tok && a && am) ? block_lists(N, block_of, Tb, start, tok) : ORC_BAD;
    for (int r = 0; r < nrows && rc == ORC_OK; ++r) {
        if (rows[r] < 0 || rows[r] >= N) { rc = ORC_BAD; break; }
        rc = attend_row(Q, K, V, d, rows[r], block_of, Tb, idx, keep, scale, start, tok, a, am,
                        O_rows + (size_t)r * d, lse_rows + r);
    }
    free(start); free(tok); free(a); free(am);
    return rc;
}

/* Joint text + image attention of one image query n (Algorithm 1: the token mask is
 * padded with ones for the T_txt text tokens, Q, K, V are the concatenations [text;
 * image], and SparseAttention runs on the whole sequence). The keys of image query n are
 * all Tt text keys (the padded columns) followed by the image keys of the kept blocks of
 * block_of[n]; scores, max, lse and the weighted sum of values are formed over that one
 * list exactly as in attend_row. */
static int attend_row_joint(const double *Q, const double *K, const double *V, int d, int n,
                            const double *Kt, const double *Vt, int Tt,
                            const int32_t *block_of, int Tb, const int32_t *idx, int keep,
                            double scale, const int *start, const int *tok, double *a, int *am,
                            double *O_row, double *lse_n)
{
    const int32_t *kept = idx + (size_t)block_of[n] * keep;
    int na = 0;
    for (int m = 0; m < Tt; ++m) {
        double dot = 0.0;
        for (int c = 0; c < d; ++c) dot += Q[(size_t)n * d + c] * Kt[(size_t)m * d + c];
        a[na] = scale * dot;
        am[na] = -1 - m;  /* text key m */
        na++;
    }
    for (int t = 0; t < keep; ++t) {
        int j = kept[t];
        if (j < 0 || j >= Tb) return ORC_BAD;
        for (int u = start[j]; u < start[j + 1]; ++u) {
            int m = tok[u];
            double dot = 0.0;
            for (int c = 0; c < d; ++c) dot += Q[(size_t)n * d + c] * K[(size_t)m * d + c];
            a[na] = scale * dot;
            am[na] = m;
            na++;
        }
    }
    double mx = -INFINITY;
    for (int u = 0; u < na; ++u) if (a[u] > mx) mx = a[u];
    double sum = 0.0;
    for (int u = 0; u < na; ++u) sum += exp(a[u] - mx);
    double l = mx + log(sum);
    *lse_n = l;
    for (int c = 0; c < d; ++c) O_row[c] = 0.0;
    for (int u = 0; u < na; ++u) {
        double p = exp(a[u] - l);
        const double *vm = am[u] >= 0 ? V + (size_t)am[u] * d : Vt + (size_t)(-1 - am[u]) * d;
        for (int c = 0; c < d; ++c) O_row[c] += p * vm[c];
    }
    return ORC_OK;
}

/* Joint attention of one slice (Algorithm 1 with its text segment, returning the image
 * rows O[T_txt:] only): Q, K, V [N][d] image tokens, Kt, Vt [Tt][d] text tokens.
 * Text queries are not evaluated: Algorithm 1 returns the image features only, so
 * their rows cannot affect the result. */
int ssba_oracle_attention_joint(const double *Q, const double *K, const double *V, int N, int d,
                                const double *Kt, const double *Vt, int Tt,
                                const int32_t *block_of, int Tb, const int32_t *idx, int keep,
                                double scale, double *O, double *lse)
{
    if (!Q || !K || !V || !block_of || !idx || !O || !lse) return ORC_BAD;
    if (N <= 0 || d <= 0 || Tb <= 0 || keep <= 0 || keep > Tb || Tt < 0) return ORC_BAD;
    if (Tt > 0 && (!Kt || !Vt)) return ORC_BAD;
    int *start = (int *)malloc(sizeof(int) * ((size_t)Tb + 1));
    int *tok = (int *)malloc(sizeof(int) * (size_t)N);
    double *a = (double *)malloc(sizeof(double) * ((size_t)N + (size_t)Tt));
    int *am = (int *)malloc(sizeof(int) * ((size_t)N + (size_t)Tt));
    int rc = (start && tok && a && am) ? block_lists(N, block_of, Tb, start, tok) : ORC_BAD;
    for (int n = 0; n < N && rc == ORC_OK; ++n)
        rc = attend_row_joint(Q, K, V, d, n, Kt, Vt, Tt, block_of, Tb, idx, keep, scale, start, tok, a, am,
                              O + (size_t)n * d, lse + n);
    free(start); free(tok); free(a); free(am);
    return rc;
}

/* Gradients of the sparse attention of one slice (the backward pass of Algorithm 1's
 * SparseAttention over the same expanded mask; the paper trains with it but does not write
 * it out, so this is the chain rule of the forward above). Given the output gradient dO:
 *   p_nm  = exp(a_nm - lse_n),  a_nm = scale * <Q_n, K_m>, over the allowed keys of n
 *   D_n   = sum_m p_nm <dO_n, V_m>  (= <dO_n, O_n>)
 *   dV_m  = sum_n p_nm dO_n
 *   ds_nm = p_nm (<dO_n, V_m> - D_n)
 *   dQ_n  = scale * sum_m ds_nm K_m,   dK_m = scale * sum_n ds_nm Q_n.
 * Every sum runs over the pairs (n, m) the mask allows; query rows in token order, keys as
 * in attend_row. */
int ssba_oracle_attention_backward(const double *Q, const double *K, const double *V, const double *dO,
                                   int N, int d, const int32_t *block_of, int Tb, const int32_t *idx,
                                   int keep, double scale, double *dQ, double *dK, double *dV)
{
    if (!Q || !K || !V || !dO || !block_of || !idx || !dQ || !dK || !dV) return ORC_BAD;
    if (N <= 0 || d <= 0 || Tb <= 0 || keep <= 0 || keep > Tb) return ORC_BAD;
    int *start = (int *)malloc(sizeof(int) * ((size_t)Tb + 1));
    int *tok = (int *)malloc(sizeof(int) * (size_t)N);
    double *a = (double *)malloc(sizeof(double) * (size_t)N);
    int *am = (int *)malloc(sizeof(int) * (size_t)N);
    double *dp = (double *)malloc(sizeof(double) * (size_t)N);
    int rc = (start && tok && a && am && dp) ? block_lists(N, block_of, Tb, start, tok) : ORC_BAD;
    if (rc == ORC_OK) {
        memset(dQ, 0, sizeof(double) * (size_t)N * d);
        memset(dK, 0, sizeof(double) * (size_t)N * d);
        memset(dV, 0, sizeof(double) * (size_t)N * d);
    }
    for (int n = 0; n < N && rc == ORC_OK; ++n) {
        const int32_t *kept = idx + (size_t)block_of[n] * keep;
        int na = 0;
        for (int t = 0; t < keep && rc == ORC_OK; ++t) {
            int j = kept[t];
            if (j < 0 || j >= Tb) { rc = ORC_BAD; break; }
            for (int u = start[j]; u < start[j + 1]; ++u) {
                int m = tok[u];
                double dot = 0.0;
                for (int c = 0; c < d; ++c) dot += Q[(size_t)n * d + c] * K[(size_t)m * d + c];
                a[na] = scale * dot;
                am[na] = m;
                na++;
            }
        }
        if (rc != ORC_OK) break;
        double mx = -INFINITY;
        for (int u = 0; u < na; ++u) if (a[u] > mx) mx = a[u];
        double sum = 0.0;
        for (int u = 0; u < na; ++u) sum += exp(a[u] - mx);
        const double lse = mx + log(sum);
        double D = 0.0;
        for (int u = 0; u < na; ++u) {
            const double *vm = V + (size_t)am[u] * d;
            double t = 0.0;
            for (int c = 0; c < d; ++c) t += dO[(size_t)n * d + c] * vm[c];
            dp[u] = t;
            D += exp(a[u] - lse) * t;
        }
        for (int u = 0; u < na; ++u) {
            const int m = am[u];
            const double p = exp(a[u] - lse);
            const double ds = p * (dp[u] - D);
            for (int c = 0; c < d; ++c) {
                dV[(size_t)m * d + c] += p * dO[(size_t)n * d + c];
                dQ[(size_t)n * d + c] += scale * ds * K[(size_t)m * d + c];
                dK[(size_t)m * d + c] += scale * ds * Q[(size_t)n * d + c];
            }
        }
    }
    free(start); free(tok); free(a); free(am); free(dp);
    return rc;
}

/* Dense softmax attention over all N keys (Table 2 "baseline 0%" sparsity). */
int ssba_oracle_dense_attention(const double *Q, const double *K, const double *V,
                                int N, int d, double scale, double *O, double *lse)
{
    if (!Q || !K || !V || !O || !lse || N <= 0 || d <= 0) return ORC_BAD;
    double *a = (double *)malloc(sizeof(double) * (size_t)N);
    if (!a) return ORC_BAD;
    for (int n = 0; n < N; ++n) {
        double mx = -INFINITY;
        for (int m = 0; m < N; ++m) {
            double dot = 0.0;
            for (int c = 0; c < d; ++c) dot += Q[(size_t)n * d + c] * K[(size_t)m * d + c];
            a[m] = scale * dot;
            if (a[m] > mx) mx = a[m];
        }
        double sum = 0.0;
        for (int m = 0; m < N; ++m) sum += exp(a[m] - mx);
        double l = mx + log(sum);
        lse[n] = l;
        for (int c = 0; c < d; ++c) O[(size_t)n * d + c] = 0.0;
        for (int m = 0; m < N; ++m) {
            double p = exp(a[m] - l);
            for (int c = 0; c < d; ++c) O[(size_t)n * d + c] += p * V[(size_t)m * d + c];
        }
    }
    free(a);
    return ORC_OK;
}

/* ---- whole-tensor drivers over [B*heads] slices --------------------------------
 * Algorithm 1 steps 2-7 for every (batch, head) slice of contiguous
 * [BH][N][d] tensors. Slices are independent, so the OpenMP loop over slices
 * does not change any result. */

int ssba_oracle_build_mask_all(const double *Q, const double *K, int BH, int H, int W,
                               int d, int blk, int shift_r, int shift_c, double rho,
                               int32_t *idx, int32_t *cnt, double *S_out)
{
    if (!Q || !K || !idx || !cnt || BH <= 0 || d <= 0 || blk <= 0) return ORC_BAD;
    if (H % blk || W % blk || rho < 0.0 || rho >= 1.0) return ORC_BAD;
    int N = H * W, Tb = N / (blk * blk);
    int k_drop = ssba_oracle_drop_count(Tb, rho), keep = Tb - k_drop;
    if (keep < 1) return ORC_BAD;
    int32_t *block_of = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    if (!block_of) return ORC_BAD;
    if (ssba_oracle_partition(H, W, blk, shift_r, shift_c, block_of) != ORC_OK) {
        free(block_of);
        return ORC_BAD;
    }
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(|:bad)
    for (int s = 0; s < BH; ++s) {
        double *qb = (double *)malloc(sizeof(double) * (size_t)Tb * d);
        double *kb = (double *)malloc(sizeof(double) * (size_t)Tb * d);
        double *S = (double *)malloc(sizeof(double) * (size_t)Tb * Tb);
        if (!qb || !kb || !S) { bad |= 1; free(qb); free(kb); free(S); continue; }
        bad |= ssba_oracle_pool(Q + (size_t)s * N * d, N, d, block_of, Tb, qb);
        bad |= ssba_oracle_pool(K + (size_t)s * N * d, N, d, block_of, Tb, kb);
        bad |= ssba_oracle_affinity(qb, kb, Tb, d, S);
        bad |= ssba_oracle_gate(S, Tb, k_drop, idx + (size_t)s * Tb * keep);
        for (int i = 0; i < Tb; ++i) cnt[(size_t)s * Tb + i] = keep;
        if (S_out) memcpy(S_out + (size_t)s * Tb * Tb, S, sizeof(double) * (size_t)Tb * Tb);
        free(qb); free(kb); free(S);
    }
    free(block_of);
    return bad ? ORC_BAD : ORC_OK;
}

int ssba_oracle_forward_all(const double *Q, const double *K, const double *V, int BH,
                            int H, int W, int d, int blk, int shift_r, int shift_c,
                            const int32_t *idx, int keep, double scale,
                            double *O, double *lse)
{
    if (!Q || !K || !V || !idx || !O || !lse || BH <= 0 || blk <= 0) return ORC_BAD;
    if (H % blk || W % blk) return ORC_BAD;
    int N = H * W, Tb = N / (blk * blk);
    int32_t *block_of = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    if (!block_of) return ORC_BAD;
    if (ssba_oracle_partition(H, W, blk, shift_r, shift_c, block_of) != ORC_OK) {
        free(block_of);
        return ORC_BAD;
    }
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(|:bad)
    for (int s = 0; s < BH; ++s) {
        size_t off = (size_t)s * N * d;
        bad |= ssba_oracle_attention(Q + off, K + off, V + off, N, d, block_of, Tb,
                                     idx + (size_t)s * Tb * keep, keep, scale,
                                     O + off, lse + (size_t)s * N);
    }
    free(block_of);
    return bad ? ORC_BAD : ORC_OK;
}

int ssba_oracle_forward_joint_all(const double *Q, const double *K, const double *V,
                                  const double *Kt, const double *Vt, int Tt, int BH,
                                  int H, int W, int d, int blk, int shift_r, int shift_c,
                                  const int32_t *idx, int keep, double scale,
                                  double *O, double *lse)
{
    if (!Q || !K || !V || !idx || !O || !lse || BH <= 0 || blk <= 0 || Tt < 0) return ORC_BAD;
    if (H % blk || W % blk) return ORC_BAD;
    int N = H * W, Tb = N / (blk * blk);
    int32_t *block_of = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    if (!block_of) return ORC_BAD;
    if (ssba_oracle_partition(H, W, blk, shift_r, shift_c, block_of) != ORC_OK) {
        free(block_of);
        return ORC_BAD;
    }
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(|:bad)
    for (int s = 0; s < BH; ++s) {
        size_t off = (size_t)s * N * d, toff = (size_t)s * Tt * d;
        bad |= ssba_oracle_attention_joint(Q + off, K + off, V + off, N, d, Tt ? Kt + toff : NULL,
                                           Tt ? Vt + toff : NULL, Tt, block_of, Tb,
                                           idx + (size_t)s * Tb * keep, keep, scale, O + off,
                                           lse + (size_t)s * N);
    }
    free(block_of);
    return bad ? ORC_BAD : ORC_OK;
}

int ssba_oracle_backward_all(const double *Q, const double *K, const double *V, const double *dO,
                             int BH, int H, int W, int d, int blk, int shift_r, int shift_c,
                             const int32_t *idx, int keep, double scale,
                             double *dQ, double *dK, double *dV)
{
    if (!Q || !K || !V || !dO || !idx || !dQ || !dK || !dV || BH <= 0 || blk <= 0) return ORC_BAD;
    if (H % blk || W % blk) return ORC_BAD;
    int N = H * W, Tb = N / (blk * blk);
    int32_t *block_of = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    if (!block_of) return ORC_BAD;
    if (ssba_oracle_partition(H, W, blk, shift_r, shift_c, block_of) != ORC_OK) {
        free(block_of);
        return ORC_BAD;
    }
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(|:bad)
    for (int s = 0; s < BH; ++s) {
        size_t off = (size_t)s * N * d;
        bad |= ssba_oracle_attention_backward(Q + off, K + off, V + off, dO + off, N, d, block_of, Tb,
                                              idx + (size_t)s * Tb * keep, keep, scale,
                                              dQ + off, dK + off, dV + off);
    }
    free(block_of);
    return bad ? ORC_BAD : ORC_OK;
}

int ssba_oracle_dense_all(const double *Q, const double *K, const double *V, int BH,
                          int N, int d, double scale, double *O, double *lse)
{
    if (BH <= 0) return ORC_BAD;
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(|:bad)
    for (int s = 0; s < BH; ++s) {
        size_t off = (size_t)s * N * d;
        bad |= ssba_oracle_dense_attention(Q + off, K + off, V + off, N, d, scale,
                                           O + off, lse + (size_t)s * N);
    }
    return bad ? ORC_BAD : ORC_OK;
}

/* Thread control for the timing leg only; results do not depend on it. */
int ssba_oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void ssba_oracle_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* ---------------------------------------------------------------- Haar wavelets (T-DVAE)
 * One level of the 2-D Haar kernel bank F = {LL, HL, LH, HH} (Sec. 2.3 DWT-Enhanced
 * Architecture), orthonormal, stride 2, per channel. x [C][H][W] (H, W even); for the 2 x 2
 * window a = x[2i][2j], b = x[2i][2j+1], c = x[2i+1][2j], d = x[2i+1][2j+1]:
 *   LL = (a + b + c + d) / 2,  HL = (a - b + c - d) / 2,
 *   LH = (a + b - c - d) / 2,  HH = (a - b - c + d) / 2.
 * y [nb * C][H/2][W/2], subband-major: bands LL, HL, LH (and HH when nb = 4) of every
 * channel; nb = 3 keeps c = {LL, HL, LH} as the paper's recursion does. */
int ssba_oracle_haar_dwt(const double *x, int C, int H, int W, int nb, double *y)
{
    if (!x || !y || C <= 0 || H <= 0 || W <= 0 || (H & 1) || (W & 1) || (nb != 3 && nb != 4)) return ORC_BAD;
    const int h2 = H / 2, w2 = W / 2;
    for (int ch = 0; ch < C; ++ch)
        for (int i = 0; i < h2; ++i)
            for (int j = 0; j < w2; ++j) {
                const double *xc = x + (size_t)ch * H * W;
                const double a = xc[(size_t)(2 * i) * W + 2 * j], b = xc[(size_t)(2 * i) * W + 2 * j + 1];
                const double c = xc[(size_t)(2 * i + 1) * W + 2 * j], d = xc[(size_t)(2 * i + 1) * W + 2 * j + 1];
                const double band[4] = {(a + b + c + d) / 2, (a - b + c - d) / 2, (a + b - c - d) / 2,
                                        (a - b - c + d) / 2};
                for (int s = 0; s < nb; ++s) y[((size_t)s * C + ch) * h2 * w2 + (size_t)i * w2 + j] = band[s];
            }
    return ORC_OK;
}

/* The inverse (the transpose of the orthonormal bank): y [nb * C][H/2][W/2] as above (HH
 * taken as 0 when nb = 3), x [C][H][W]:
 *   a = (LL + HL + LH + HH) / 2,  b = (LL - HL + LH - HH) / 2,
 *   c = (LL + HL - LH - HH) / 2,  d = (LL - HL - LH + HH) / 2. */
int ssba_oracle_haar_iwt(const double *y, int C, int H, int W, int nb, double *x)
{
    if (!x || !y || C <= 0 || H <= 0 || W <= 0 || (H & 1) || (W & 1) || (nb != 3 && nb != 4)) return ORC_BAD;
    const int h2 = H / 2, w2 = W / 2;
    for (int ch = 0; ch < C; ++ch)
        for (int i = 0; i < h2; ++i)
            for (int j = 0; j < w2; ++j) {
                double v[4] = {0, 0, 0, 0};
                for (int s = 0; s < nb; ++s) v[s] = y[((size_t)s * C + ch) * h2 * w2 + (size_t)i * w2 + j];
                const double LL = v[0], HL = v[1], LH = v[2], HH = v[3];
                double *xc = x + (size_t)ch * H * W;
                xc[(size_t)(2 * i) * W + 2 * j] = (LL + HL + LH + HH) / 2;
                xc[(size_t)(2 * i) * W + 2 * j + 1] = (LL - HL + LH - HH) / 2;
                xc[(size_t)(2 * i + 1) * W + 2 * j] = (LL + HL - LH - HH) / 2;
                xc[(size_t)(2 * i + 1) * W + 2 * j + 1] = (LL - HL - LH + HH) / 2;
            }
    return ORC_OK;
}
