// Launch interface of the tcgen05 projection GEMMs (gemm_tc.cu).
#pragma once

#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.h"

namespace fsx {

constexpr int kTcTileRows = 128;  // weight rows per tile
constexpr int kTcTileK = 64;      // K per tile
constexpr int kTcTileBytes = kTcTileRows * kTcTileK * 2;

struct TcGemmArgs {
  const unsigned char* w;  // packed tiles: tile (n_tile, k_tile) at (n_tile * K/64 + k_tile) * 16 KB
  int N;                   // weight rows (multiple of 128)
  int K;                   // reduction length (multiple of 64)
  int M;                   // tokens
  __half* y;               // kEpiStore: y[m, n]; kEpiSwiglu: y[m, n / 2]
  int ldy;
  float* xo;               // kEpiResidual: xo[m, n] += result, xo16 = fp16 copy
  __half* xo16;
  int ldxo;
  // sums of x^2 per token over 128-column groups: [n_ss][ss_stride], group j = columns 128j..128j+127.
  // kEpiResidual writes group blockIdx.x of the updated rows; RMSNorm-fused GEMMs read all groups.
  float* ss_out;
  const float* ss_in;
  int n_ss;
  int ss_stride;
  int* status;
  // split K (kEpiResidual only): k_splits > 1 cuts each tile's K steps into k_splits
  // near-equal ranges run by different CTAs (never more units than SMs, one CTA per
  // SM, so all are resident); each writes its fp32 partial tile to `part`
  // ([tile][split][BN tokens][128]), waits until the tile's k_splits partials are
  // there (tile_count[tile], zero between launches), and adds them in split order
  // for its 1/k_splits share of the tile's tokens.
  int k_splits;
  float* part;
  int* tile_count;
  // pair variant: index of the tile at `w` in the weight map (tiles of 16 KB from the map's base)
  int w_tile0;
};

// k splits for a residual GEMM with `tiles` output tiles of KT k steps on `sm_count` SMs
int gemm_tc_k_splits(int tiles, int KT, int sm_count);
// bytes of the split-K partial workspace that covers every GEMM of a handle
size_t gemm_tc_part_bytes(int sm_count);

cudaError_t gemm_tc_set_attributes();
// co-resident CTA pairs of the pair variant on this device (0: the variant is not available)
int gemm_tc_pair_clusters();
// map_w != nullptr selects the pair variant (bn 256, RMSNorm-fused store epilogue, N a multiple
// of 256, no K split): map_a then has 128-row boxes and map_w covers the packed weight tiles
cudaError_t launch_gemm_tc(const CUtensorMap& map_a, const TcGemmArgs& args, int bn, int epi, bool norm,
                           cudaStream_t stream, bool pdl, const CUtensorMap* map_w = nullptr);
// rows[128]: pointers to the 128 source rows (fp32, length >= k0 + 64); col_scale: optional per-K gain.
void pack_tc_tile(const float* const* rows, const float* col_scale, int k0, __half* out);
// 2-D fp16 tensor map over a row-major [rows, cols] buffer with a (box_rows x 64) box and 128-byte swizzle.
bool encode_act_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows);
// 3-D bf16 tensor map over a token-major KV cache [rows, n_heads, 128]: a box is 64 tokens of one
// head and 64 of its 128 dims, 128-byte swizzle (the attention's operand layout).
bool encode_cache_map(CUtensorMap* map, const void* base, uint64_t rows, uint32_t n_heads);
// 2-D fp16 tensor map over an output y[rows, cols] with row stride `ld` elements, 64-column x
// 32-row boxes, 128-byte swizzle (the store / SwiGLU epilogues' TMA stores)
bool encode_out_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t ld);
// 3-D fp16 tensor map over `n_tiles` packed 16 KB weight tiles [tiles][128 rows][64], no swizzle:
// a box is one whole tile image
bool encode_weight_map(CUtensorMap* map, const void* base, uint64_t n_tiles);

}  // namespace fsx
