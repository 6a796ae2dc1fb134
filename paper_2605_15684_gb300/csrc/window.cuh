// window.cuh -- a shifted 8x8 window of the token grid as TMA boxes (Sec. 2.2: the shifted
// windows are the blocks; the shift is index arithmetic, nothing is rolled). For block 8 and a
// shift that is a multiple of 4 tokens, a window either lies inside the grid (one 8x8 box) or
// is cut 4 + 4 by the grid edge (two or four boxes); the 8 KB bf16 tile then holds the boxes
// one after the other, and tile_row_pos gives the in-window position of each tile row.
#pragma once

#include <cuda.h>

#include "common.cuh"
#include "ptx.cuh"

namespace ssba {
namespace win {

// Tensor-map box shapes (d x cols x rows), in the order of the maps encode_window_maps writes.
enum BoxShape { kBox8x8 = 0, kBox8c4r = 1, kBox4c8r = 2, kBox4x4 = 3 };

// Origin (row, col) of the shifted 8x8 window `label` in the unshifted grid. With block
// 8 and a shift that is a multiple of 4, a window either fits (origin <= size - 8) or is
// split 4 + 4 by the grid edge (origin = size - 4).
__device__ __forceinline__ void window_origin(const Grid& g, int label, int& r0, int& c0)
{
    const int br = label / g.bw, bc = label - br * g.bw;
    r0 = br * 8 - g.sr;
    if (r0 < 0) r0 += g.H;
    c0 = bc * 8 - g.sc;
    if (c0 < 0) c0 += g.W;
}

// Window of `label` packed in one word: origin row r0 (bits 0-14), origin column c0 (bits
// 15-29) and the box shape class (bits 30-31: 0 one 8x8 box, 1 split rows, 2 split columns,
// 3 both). Tabulated per CTA at kernel start, so that the producers' per-copy work is a
// shared-memory load and a switch (the producers' issue loop is on the critical path).
__device__ __forceinline__ uint32_t window_entry(const Grid& g, int label)
{
    int r0, c0;
    window_origin(g, label, r0, c0);
    const uint32_t wr = r0 + 8 > g.H, wc = c0 + 8 > g.W;
    return (uint32_t)r0 | ((uint32_t)c0 << 15) | ((wr | (wc << 1)) << 30);
}

// TMA copies of a window given its packed entry (see window_boxes).
__device__ __forceinline__ void window_boxes_e(const CUtensorMap* m4, uint32_t dst, uint32_t bar, uint32_t e, int bh)
{
    const int r0 = e & 0x7fff, c0 = (e >> 15) & 0x7fff;
    switch (e >> 30) {
        case 0:
            ptx::tma_load_4d(dst, &m4[kBox8x8], bar, 0, c0, r0, bh);
            break;
        case 1:
            ptx::tma_load_4d(dst, &m4[kBox8c4r], bar, 0, c0, r0, bh);
            ptx::tma_load_4d(dst + 4096, &m4[kBox8c4r], bar, 0, c0, 0, bh);
            break;
        case 2:
            ptx::tma_load_4d(dst, &m4[kBox4c8r], bar, 0, c0, r0, bh);
            ptx::tma_load_4d(dst + 4096, &m4[kBox4c8r], bar, 0, 0, r0, bh);
            break;
        default:
            ptx::tma_load_4d(dst, &m4[kBox4x4], bar, 0, c0, r0, bh);
            ptx::tma_load_4d(dst + 2048, &m4[kBox4x4], bar, 0, 0, r0, bh);
            ptx::tma_load_4d(dst + 4096, &m4[kBox4x4], bar, 0, c0, 0, bh);
            ptx::tma_load_4d(dst + 6144, &m4[kBox4x4], bar, 0, 0, 0, bh);
            break;
    }
}

// A window is one 8x8 box when it does not cross the grid edge, else two 8-col x 4-row boxes
// (split rows), two 4-col x 8-row boxes (split columns) or four 4x4 boxes; the tile row
// order is set by the shape class and decoded by tile_row_pos(); K and V of one label
// always share it.
// Tile row r of window `label` -> in-window position (row-major over the 8x8 window).
__device__ __forceinline__ int tile_row_pos(const Grid& g, int label, int r)
{
    int r0, c0;
    window_origin(g, label, r0, c0);
    const bool wr = r0 + 8 > g.H, wc = c0 + 8 > g.W;
    if (!wc) return r;  // 8-wide rows, row-major (one box or two row halves)
    if (!wr) {          // two 8x4 column halves
        const int h = r >> 5, a = (r >> 2) & 7, b = r & 3;
        return a * 8 + 4 * h + b;
    }
    const int q = r >> 4, a = (r >> 2) & 3, b = r & 3;  // four 4x4 quadrants
    return (4 * (q >> 1) + a) * 8 + 4 * (q & 1) + b;
}

// Inverse of tile_row_pos: the tile row that holds in-window position pos of block `label`.
__device__ __forceinline__ int tile_row_of(const Grid& g, int label, int pos)
{
    int r0, c0;
    window_origin(g, label, r0, c0);
    const bool wr = r0 + 8 > g.H, wc = c0 + 8 > g.W;
    if (!wc) return pos;
    const int a = pos >> 3, c = pos & 7;
    if (!wr) return (c >> 2) * 32 + a * 4 + (c & 3);
    return ((a >> 2) * 2 + (c >> 2)) * 16 + (a & 3) * 4 + (c & 3);
}

// Block label and in-window position of token t (the inverse of Grid::token).
__device__ __forceinline__ void token_block(const Grid& g, int t, int& label, int& pos)
{
    const int r = t / g.W, c = t - r * g.W;
    int R = r + g.sr, C = c + g.sc;
    R -= R >= g.H ? g.H : 0;
    C -= C >= g.W ? g.W : 0;
    label = (R >> 3) * g.bw + (C >> 3);
    pos = (R & 7) * 8 + (C & 7);
}

}  // namespace win

// [B*heads][H][W][64] bf16 viewed as 4-D tensor maps, one per box shape (BoxShape order),
// 128-byte swizzle. False when the driver's encoder is unavailable or refuses the layout.
bool encode_window_maps(CUtensorMap* m4, const void* base, int BH, int H, int W);

}  // namespace ssba
