// Internal launch interface between the C-ABI host code (fsx.cu) and the
// kernel translation units. Not part of the public ABI.
#pragma once

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
  const void* frames;
  float* waypoints;
};

// ------------------------------------------------------------------ GEMM
// Y[M, N] = A[M, K] . W[N, K]^T with W packed as 16x16 fp16 fragment blocks.
enum GemmPrologue { kProNorm = 0, kProCopy = 1 };
enum GemmEpilogue { kEpiStore = 0, kEpiResidual = 1, kEpiSwiglu = 2 };

struct GemmArgs {
  const uint4* w;      // packed weights: block (nb, kb) = 32 x uint4 at (nb * K/16 + kb) * 32
  int n_rows;          // packed rows N (multiple of 16)
  int K;               // reduction length (multiple of 64)
  int ks;              // K per split (multiple of 64); the last split may be shorter
  int M;               // activation rows
  int m_tiles_per_cta; // 48-row tiles per CTA along grid.z
  // prologue kProNorm: A = fp16 copy of the residual stream (rows of length K);
  // the norm gain is folded into w and the epilogue scales by the row's 1/rms
  const __half* x16;
  int ldx16;
  // prologue kProCopy: A = fp16 rows
  const __half* a;
  int lda;
  // epilogue kEpiStore: y[m, n] fp16; kEpiSwiglu: y[m, n/2] = silu(gate) * up fp16
  __half* y;
  int ldy;
  // epilogue kEpiResidual: xo[m, n] += sum over the K splits (one cluster), fp32,
  // and xo16[m, n] = fp16 copy of the updated value
  float* xo;
  __half* xo16;
  int ldxo;
  int* status;
};

struct GemmPlan {
  int nb;       // 16-row blocks per CTA (1 or 2)
  int ks;
  int prologue;
  int epilogue;
  dim3 grid;
  size_t smem;
};

GemmPlan plan_gemm(int n_rows, int K, int M, int nb, int ks, int prologue, int epilogue, int sm_count);
cudaError_t launch_gemm(const GemmPlan& plan, const GemmArgs& args, cudaStream_t stream, bool pdl);
cudaError_t gemm_set_attributes();

// ------------------------------------------------------------- attention
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
  int* status;
};

size_t attention_workspace_bytes(int B, int n_heads, int n_splits);
cudaError_t launch_attention(const AttnArgs& a, int B, int cache_dtype, cudaStream_t stream, bool pdl);
cudaError_t attention_set_attributes();
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

// Launch helper: cudaLaunchKernelEx with the programmatic-stream-serialisation
// attribute when `pdl` is set and a (cluster_x, cluster_y, 1) cluster when either exceeds 1.
cudaError_t launch_ex(const void* fn, dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                      bool pdl, void** args, int cluster_y = 1, int cluster_x = 1);

}  // namespace fsx
