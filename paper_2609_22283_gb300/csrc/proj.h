// Launch parameters of the QKV projection kernel (qkv_gemm.cu), apart from
// the attention and RoPE declarations in internal.h.
#pragma once

#include "internal.h"

namespace sva {

// The QKV projection y = x W^T + b split into q, k, v (sva_qkv_project).
struct ProjParams {
  CUtensorMap tmap_x;   // x as 2D (C, rows), box (64, 128), 128B swizzle
  CUtensorMap tmap_w;   // weight as 2D (C, 3N), box (64, BN / 2): one CTA's half of a tile
  CUtensorMap tmap_wh;  // the same weight with box (64, BN / 4): half-width items
  // out[i] as 2D (N, rows), box (32, 32), 64B swizzle: the epilogue's tile
  // stores.  With rope_on: tmap_out[0] is Q' token-major, tmap_out[1] the
  // slot pool as 3D (d, T, num_slots * 2 * H) with the (slot, K|V, head)
  // stride Tpad * d, box (32, 32, 1), so that rows past T are not written.
  CUtensorMap tmap_out[3];
  const float* bias;    // [3N] fp32, or null
  void* out[3];         // q, k, v: bf16 [rows][N]
  int* status;          // device status word
  int32_t rows, C, N;   // N = H * d outputs per tensor
  int32_t n_mtiles, n_ntiles, n_kblocks;  // 256-row tiles, BN-column tiles, 64-wide K blocks
  // Work items: output tiles 0..n_whole-1 whole (tile t in the grouped raster
  // of the kernel: groups of 16 row tiles, row tile fastest); the tiles
  // n_whole.. as two half-width items each (columns [0, BN/2) and [BN/2, BN)
  // of the tile), items n_whole.. n_items-1.
  int32_t n_items, n_whole;
  uint64_t timeout_ns;
  // Fused RoPE + cache scatter epilogue (sva_qkv_project_rope): q and k are
  // rotated in fp32 before their one bf16 rounding, Q' goes to out[0], K' and
  // V into the nodes' own slots (rope.cache, rope.nodes); out[1], out[2] and
  // rope.k_new / v_new / q are unused; rope.tab_h and rope.tab_w point at the
  // pair-major copies of those tables.  rows = rope.n_nodes * rope.T.
  int32_t rope_on;
  RopeParams rope;
};

// `grid` CTAs in clusters of two (grid even): each pair computes 256-row
// tiles with two-SM MMAs.
cudaError_t launch_qkv_project(const ProjParams& p, int block_n, int grid, cudaStream_t s);

// Clusters of two CTAs of the projection kernel that can be resident at once
// on the current device (one CTA per SM): the persistent grid's pair count.
cudaError_t qkv_project_max_pairs(int block_n, int* pairs);

}  // namespace sva
