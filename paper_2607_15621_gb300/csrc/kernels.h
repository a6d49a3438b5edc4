// Internal launch interface between the C-ABI host code (fsx.cu) and the
// kernel translation units. Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace fsx {

constexpr int kMaxLayers = 128;
constexpr int kTokTile = 48;    // token rows per tensor-core tile (6 x n8)
constexpr int kHeadDim = 128;   // backbone head width the kernels are built for
constexpr int kMaxSplits = 64;

// Per-tick pointers, uploaded to device memory when they change so that the
// captured graph stays valid across ticks with different caller buffers.
struct TickArgs {
  const void* k_cache[kMaxLayers];
  const void* v_cache[kMaxLayers];
  const int64_t* offsets;
  // optional [B]: first cache row of vehicle b; its rows are then starts[b] ..
  // starts[b] + (offsets[b+1] - offsets[b]) - 1, and the ranges of different
  // vehicles may overlap or leave gaps (offsets then only give the lengths)
  const int64_t* starts;
  const void* frames;
  float* waypoints;
};

// ------------------------------------------------------------ epilogues
// Epilogues of the tensor-core projection GEMMs (gemm_tc.cu).
enum GemmEpilogue { kEpiStore = 0, kEpiResidual = 1, kEpiSwiglu = 2 };

// ------------------------------------------------------------- attention
// Entry z of the batched tick's attention schedule (written by the embed kernel in
// longest-cache-first order): vehicle b, its first cache row and its number of rows.
struct AttnPlan {
  long long lo;
  int b;
  int len;  // -1 when the caller's offsets give no valid length
};

struct AttnArgs {
  const __half* q;
  long long q_stride;
  const __half* k_own;
  const __half* v_own;
  long long own_stride;
  int n_q;
  int n_own;
  const void* k_cache;        // used when targs == nullptr
  const void* v_cache;
  const TickArgs* targs;      // device tick arguments (cache pointers of `layer`)
  int layer;
  const int64_t* offsets;     // used when targs == nullptr
  long long max_total;        // offsets[B] bound (checked on the device)
  int n_heads;
  int n_splits;
  __half* out;                // [B*n_q, out_stride]
  long long out_stride;
  float* lse;                 // optional [B, H, n_q] natural log
  float* part_o;              // [B, H, S, 48, 128] when n_splits > 1
  float* part_lse;            // [B, H, S, 48]   (log2 domain)
  const int* order;           // optional [B]: CTA row z works on vehicle order[z] (longest cache first)
  const AttnPlan* plan;       // optional [B] (tensor-core path): CTA row z works on plan[z]
  // optional (tensor-core path, with targs): [2 n_layers] TMA maps of the layers' K and V caches
  // (bf16 [rows, n_heads, 128]); whole 64-key chunks are then loaded by TMA
  const CUtensorMap* cache_maps;
  int* status;
};

size_t attention_workspace_bytes(int B, int n_heads, int n_splits);
cudaError_t launch_attention(const AttnArgs& a, int B, int cache_dtype, cudaStream_t stream, bool pdl);
cudaError_t attention_set_attributes();
// tcgen05 path: bf16 cache, one split, n_q <= 48, 1 <= n_own <= 64
bool attention_tc_eligible(const AttnArgs& a, int cache_dtype);
cudaError_t launch_attention_tc(const AttnArgs& a, int B, cudaStream_t stream, bool pdl);
cudaError_t attention_tc_set_attributes();
int attention_launch_count(int n_splits);

// --------------------------------------------------------- embed / head
struct EmbedArgs {
  const float* act_emb;   // [n_action, d]
  const float* pos_emb;   // [T, d]
  const TickArgs* targs;  // frames + offsets
  int frame_dtype;
  int n_action, n_frame, d;
  int B;
  long long max_total;
  float* x;               // [B*T, d]
  __half* x16;            // fp16 copy of x
  float* ss;              // per-row sums of x^2 over 128-column groups, [d/128][ss_stride]
  int ss_stride;
  int* order;             // optional [B]: vehicles by decreasing cache length (ties by index)
  AttnPlan* plan;         // optional [B]: the same order with each vehicle's cache range
  int* status;
};
cudaError_t launch_embed(const EmbedArgs& a, cudaStream_t stream, bool pdl);

struct HeadArgs {
  const float* x;
  const float* final_norm;
  const float* head_w;
  const float* head_b;
  const TickArgs* targs;  // waypoint output pointer
  float* out;             // used when targs == nullptr
  int d, T, n_waypoints, B;
  int* status;
};
cudaError_t launch_head(const HeadArgs& a, cudaStream_t stream, bool pdl);

// Two-layer waypoint head of the ten-token layout (Sec. 3.1): waypoint j of vehicle b =
// W_h2 silu(W_h1 RMSNorm(x_{b,j}; g_f) + b_h1) + b_h2, read from token row j of the vehicle.
struct Head2Args {
  const float* x;          // token row j of vehicle b at x + (b * vehicle_rows + j) * d
  long long vehicle_rows;  // token rows per vehicle in x
  const float* final_norm; // [d]
  const float* w;          // W_h1 [d, d], b_h1 [d], W_h2 [2, d], b_h2 [2], fp32 row-major [out, in]
  const TickArgs* targs;   // waypoint output pointer
  int d, n_waypoints, B;
  int* status;             // no waypoint is written when it is set
};
cudaError_t launch_head2(const Head2Args& a, cudaStream_t stream, bool pdl);

// State token and visual tokens of the ten-token layout into a tick's fp32 frame rows:
// frames[b, 0] = W_s2 silu(W_s1 state_b + b_s1) + b_s2, frames[b, 1 + i] = visual[b, i].
struct StateArgs {
  const float* state;      // [B, 16]
  const void* visual;      // [B, 4, d] of visual_dtype (fsx_dtype)
  int visual_dtype;
  const float* w;          // W_s1 [d, 16], b_s1 [d], W_s2 [d, d], b_s2 [d]
  float* frames;           // [B, 5, d]
  int d, B;
};
cudaError_t launch_state_tokens(const StateArgs& a, cudaStream_t stream);

// Launch helper: cudaLaunchKernelEx with the programmatic-stream-serialisation
// attribute when `pdl` is set and a (cluster_x, cluster_y, 1) cluster when either exceeds 1.
cudaError_t launch_ex(const void* fn, dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                      bool pdl, void** args, int cluster_y = 1, int cluster_x = 1);

}  // namespace fsx
