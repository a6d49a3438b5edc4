// The paper's own ten-token layout of the action expert (Sec. 3.1): per vehicle and
// frame, one state token -- a two-layer MLP of the 16 ego-state values (previous five
// waypoints, control triplet, speed, target point) -- the frame's four visual tokens
// and five learned waypoint queries; after the shared layer stack a two-layer head
// decodes each query token into one (x, y) waypoint.
//
// The layer stack is the tick of fsx.cu unchanged: its own keys are attended
// bidirectionally with learned positions and no rotary phase, so the order in which
// the ten tokens are held does not change the result once the position table follows
// them. The handle therefore holds the queries as its five learned action tokens
// (rows 0-4, read by the head) and the state token plus the four visual tokens as its
// five frame rows (rows 5-9), with the paper's position rows permuted to that order.
// Per tick: state_tokens_kernel writes [state token ; visual tokens] of every
// vehicle into a handle-owned fp32 frame buffer, the tick runs on it, and
// head2_kernel (in place of the single-layer head) decodes the queries.
#include <cuda_runtime.h>

#include <cstdio>
#include <cstring>
#include <vector>

#include "../../include/fsx.h"
#include "device_util.cuh"
#include "kernels.h"

namespace fsx {

void set_error_message(const char* msg);
// hooks into the tick handle (fsx.cu)
fsx_status paper_attach(fsx_handle h, float* d_params, const float* d_head, float* d_frames, const float* d_state_w,
                        int visual_dtype);
float* paper_frames(fsx_handle h);
const float* paper_state_weights(fsx_handle h);
cudaError_t paper_order_after_last_tick(fsx_handle h, cudaStream_t st);
int paper_device(fsx_handle h);
int paper_max_batch(fsx_handle h);
int paper_d(fsx_handle h);
int paper_visual_dtype(fsx_handle h);

namespace {

constexpr int kStateDim = 16;
constexpr int kVisual = 4;
constexpr int kQueries = 5;

__device__ __forceinline__ float silu(float z) { return z / (1.f + expf(-z)); }

// y[r] = act(W[r, :] . x + bias[r]) for r < d_out, x in shared memory, d_in a multiple of
// 128 (<= 1024). Each warp takes four rows at a time and issues all of their 16-byte
// weight loads before the first multiply, so a block keeps many row loads in flight.
template <bool kSilu>
__device__ __forceinline__ void block_gemv(const float* __restrict__ W, const float* __restrict__ bias, const float* x,
                                           float* y, int d_out, int d_in) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, n_warps = blockDim.x >> 5;
  const int nk = d_in / 128;
  for (int r0 = warp * 4; r0 < d_out; r0 += n_warps * 4) {
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
    for (int kq = 0; kq < nk; ++kq) {
      const int k = kq * 128 + lane * 4;
      const float4 xv = *reinterpret_cast<const float4*>(x + k);
      float4 wv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i)
        wv[i] = r0 + i < d_out ? __ldg(reinterpret_cast<const float4*>(W + static_cast<size_t>(r0 + i) * d_in + k))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int i = 0; i < 4; ++i) acc[i] += wv[i].x * xv.x + wv[i].y * xv.y + wv[i].z * xv.z + wv[i].w * xv.w;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float v = warp_sum(acc[i]);
      if (lane == 0 && r0 + i < d_out) y[r0 + i] = kSilu ? silu(v + bias[r0 + i]) : v + bias[r0 + i];
    }
  }
}

// One block per vehicle: frames[b] = [W_s2 silu(W_s1 s_b + b_s1) + b_s2 ; visual[b, 0..3]].
// Layout of w: W_s1 [d, 16], b_s1 [d], W_s2 [d, d], b_s2 [d] (fp32, row-major [out, in]).
__global__ void state_tokens_kernel(const StateArgs a) {
  extern __shared__ float sm[];
  float* s = sm;               // [16]
  float* h1 = sm + kStateDim;  // [d]
  const int b = blockIdx.x;
  const int d = a.d;
  const float* w1 = a.w;
  const float* b1 = w1 + static_cast<size_t>(d) * kStateDim;
  const float* w2 = b1 + d;
  const float* b2 = w2 + static_cast<size_t>(d) * d;
  if (threadIdx.x < kStateDim) s[threadIdx.x] = a.state[static_cast<size_t>(b) * kStateDim + threadIdx.x];
  __syncthreads();
  for (int o = threadIdx.x; o < d; o += blockDim.x) {
    float acc = b1[o];
#pragma unroll
    for (int k = 0; k < kStateDim; ++k) acc += w1[static_cast<size_t>(o) * kStateDim + k] * s[k];
    h1[o] = silu(acc);
  }
  __syncthreads();
  float* out = a.frames + static_cast<size_t>(b) * (1 + kVisual) * d;
  block_gemv<false>(w2, b2, h1, out, d, d);
  for (int i = threadIdx.x; i < kVisual * d; i += blockDim.x) {
    const size_t src = static_cast<size_t>(b) * kVisual * d + i;
    out[d + i] = a.visual_dtype == 1 ? __bfloat162float(static_cast<const __nv_bfloat16*>(a.visual)[src])
                                     : static_cast<const float*>(a.visual)[src];
  }
}

}  // namespace

// One block per (vehicle, waypoint): w = W_h2 silu(W_h1 RMSNorm(x; g_f) + b_h1) + b_h2
// over the query token's final state. Layout of a.w: W_h1 [d, d], b_h1 [d], W_h2 [2, d], b_h2 [2].
__global__ void head2_kernel(const Head2Args a) {
  pdl_launch_dependents();
  pdl_wait();
  if (*reinterpret_cast<volatile int*>(a.status) != 0) return;  // a device-side error: no waypoint
  extern __shared__ float sm[];
  const int d = a.d;
  float* n = sm;       // [d]
  float* h1 = sm + d;  // [d]
  __shared__ float red[32];
  __shared__ float s_rstd;
  const int b = blockIdx.x, j = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, n_warps = blockDim.x >> 5;
  const float* xr = a.x + (static_cast<size_t>(b) * a.vehicle_rows + j) * d;
  float ss = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const float v = __ldcg(xr + c);
    ss += v * v;
  }
  ss = warp_sum(ss);
  if (lane == 0) red[warp] = ss;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < n_warps; ++w) t += red[w];
    s_rstd = rsqrtf(t / static_cast<float>(d) + 1e-6f);
  }
  __syncthreads();
  const float rstd = s_rstd;
  for (int c = threadIdx.x; c < d; c += blockDim.x) n[c] = __ldcg(xr + c) * rstd * a.final_norm[c];
  __syncthreads();
  const float* w1 = a.w;
  const float* b1 = w1 + static_cast<size_t>(d) * d;
  const float* w2 = b1 + d;
  const float* b2 = w2 + static_cast<size_t>(2) * d;
  block_gemv<true>(w1, b1, n, h1, d, d);
  __syncthreads();
  float* out = a.targs->waypoints + (static_cast<size_t>(b) * a.n_waypoints + j) * 2;
  block_gemv<false>(w2, b2, h1, out, 2, d);
}

cudaError_t launch_state_tokens(const StateArgs& a_in, cudaStream_t stream) {
  StateArgs a = a_in;
  void* kargs[] = {&a};
  return launch_ex(reinterpret_cast<const void*>(&state_tokens_kernel), dim3(a.B), dim3(1024),
                   (kStateDim + a.d) * sizeof(float), stream, false, kargs);
}

cudaError_t launch_head2(const Head2Args& a_in, cudaStream_t stream, bool pdl) {
  Head2Args a = a_in;
  void* kargs[] = {&a};
  return launch_ex(reinterpret_cast<const void*>(&head2_kernel), dim3(a.B, a.n_waypoints), dim3(1024),
                   2 * a.d * sizeof(float), stream, pdl, kargs);
}

}  // namespace fsx

namespace {

fsx_status pfail(fsx_status s, const char* msg) {
  fsx::set_error_message(msg);
  return s;
}

}  // namespace

extern "C" {

fsx_status fsx_paper_create(const fsx_config* cfg, const fsx_paper_weights* w, int device, fsx_handle* out) {
  fsx::set_error_message("");
  if (!out) return pfail(FSX_ERR_INVALID_ARG, "out handle pointer is NULL");
  *out = nullptr;
  if (!cfg || !w) return pfail(FSX_ERR_INVALID_ARG, "config or weights is NULL");
  if (!w->state_w1 || !w->state_b1 || !w->state_w2 || !w->state_b2 || !w->query_emb || !w->pos_emb ||
      !w->head_w1 || !w->head_b1 || !w->head_w2 || !w->head_b2 || !w->final_norm)
    return pfail(FSX_ERR_INVALID_ARG, "a weight pointer is NULL");
  const int d = cfg->d_model;
  if (d <= 0 || d > 1024) return pfail(FSX_ERR_UNSUPPORTED, "d_model must be in 1..1024");
  fsx_config c = *cfg;
  c.n_action = fsx::kQueries;      // the five waypoint queries: the handle's action tokens 0-4
  c.n_frame = 1 + fsx::kVisual;    // the state token and the four visual tokens
  c.n_waypoints = fsx::kQueries;
  c.frame_dtype = FSX_F32;         // the frame rows are assembled in fp32 on the device
  const int paper_visual_dtype = cfg->frame_dtype;
  if (paper_visual_dtype != FSX_F32 && paper_visual_dtype != FSX_BF16)
    return pfail(FSX_ERR_INVALID_ARG, "frame_dtype (of the visual tokens) must be FSX_F32 or FSX_BF16");
  // position rows in the handle's token order: queries 0-4, state, visual 0-3 (paper order:
  // state, visual 0-3, queries 0-4)
  std::vector<float> pos(static_cast<size_t>(10) * d);
  for (int i = 0; i < 10; ++i) {
    const int paper_row = i < 5 ? 5 + i : i - 5;
    std::memcpy(&pos[static_cast<size_t>(i) * d], w->pos_emb + static_cast<size_t>(paper_row) * d, d * sizeof(float));
  }
  std::vector<float> zero_head(static_cast<size_t>(2) * d + 2, 0.f);  // the single-layer head is not used
  fsx_weights tw{};
  tw.act_emb = w->query_emb;
  tw.pos_emb = pos.data();
  tw.attn_norm = w->attn_norm;
  tw.wq = w->wq;
  tw.wk = w->wk;
  tw.wv = w->wv;
  tw.wo = w->wo;
  tw.mlp_norm = w->mlp_norm;
  tw.w_gate = w->w_gate;
  tw.w_up = w->w_up;
  tw.w_down = w->w_down;
  tw.final_norm = w->final_norm;
  tw.head_w = zero_head.data();
  tw.head_b = zero_head.data() + 2 * d;
  fsx_handle h = nullptr;
  fsx_status s = fsx_create(&c, &tw, device, &h);
  if (s != FSX_OK) return s;
  // device copies: head [W_h1; b_h1; W_h2; b_h2], state MLP [W_s1; b_s1; W_s2; b_s2], frame rows
  const size_t n_head = (static_cast<size_t>(d) * d + d + 2 * static_cast<size_t>(d) + 2 + 3) / 4 * 4;  // 16-byte multiple
  const size_t n_state = static_cast<size_t>(d) * fsx::kStateDim + d + static_cast<size_t>(d) * d + d;
  std::vector<float> host(n_head + n_state, 0.f);
  float* p = host.data();
  auto put = [&](const float* src, size_t n) {
    std::memcpy(p, src, n * sizeof(float));
    p += n;
  };
  put(w->head_w1, static_cast<size_t>(d) * d);
  put(w->head_b1, d);
  put(w->head_w2, 2 * static_cast<size_t>(d));
  put(w->head_b2, 2);
  p = host.data() + n_head;
  put(w->state_w1, static_cast<size_t>(d) * fsx::kStateDim);
  put(w->state_b1, d);
  put(w->state_w2, static_cast<size_t>(d) * d);
  put(w->state_b2, d);
  float* dparams = nullptr;
  float* dframes = nullptr;
  cudaError_t e = cudaSetDevice(device);
  if (e == cudaSuccess) e = cudaMalloc(&dparams, host.size() * sizeof(float));
  if (e == cudaSuccess) e = cudaMemcpy(dparams, host.data(), host.size() * sizeof(float), cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMalloc(&dframes, static_cast<size_t>(cfg->max_batch) * (1 + fsx::kVisual) * d * sizeof(float));
  if (e != cudaSuccess) {
    if (dparams) cudaFree(dparams);
    if (dframes) cudaFree(dframes);
    fsx_destroy(h);
    return pfail(e == cudaErrorMemoryAllocation ? FSX_ERR_OOM : FSX_ERR_CUDA, cudaGetErrorString(e));
  }
  s = fsx::paper_attach(h, dparams, dparams, dframes, dparams + n_head, paper_visual_dtype);
  if (s != FSX_OK) {
    cudaFree(dparams);
    cudaFree(dframes);
    fsx_destroy(h);
    return s;
  }
  *out = h;
  return FSX_OK;
}

fsx_status fsx_paper_tick(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                          const int64_t* d_offsets, int B, const void* d_visual, const float* d_state,
                          float* d_waypoints, void* stream) {
  fsx::set_error_message("");
  if (!h) return pfail(FSX_ERR_INVALID_ARG, "handle is NULL");
  if (!fsx::paper_frames(h)) return pfail(FSX_ERR_INVALID_ARG, "handle was not created by fsx_paper_create");
  if (!d_visual || !d_state) return pfail(FSX_ERR_INVALID_ARG, "visual tokens or state is NULL");
  if (B < 1 || B > fsx::paper_max_batch(h)) return pfail(FSX_ERR_INVALID_ARG, "B outside 1..max_batch");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaSetDevice(fsx::paper_device(h));
  if (e == cudaSuccess) e = fsx::paper_order_after_last_tick(h, st);
  fsx::StateArgs a{};
  a.state = d_state;
  a.visual = d_visual;
  a.visual_dtype = fsx::paper_visual_dtype(h);
  a.w = fsx::paper_state_weights(h);
  a.frames = fsx::paper_frames(h);
  a.d = fsx::paper_d(h);
  a.B = B;
  if (e == cudaSuccess) e = fsx::launch_state_tokens(a, st);
  if (e != cudaSuccess) return pfail(FSX_ERR_CUDA, cudaGetErrorString(e));
  return fsx_tick(h, k_cache, v_cache, d_offsets, B, fsx::paper_frames(h), d_waypoints, stream);
}

}  // extern "C"
