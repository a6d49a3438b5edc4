// Incremental backbone cache append (Sec. 1, Sec. 3.3): the slow system's
// forward of one frame's n_new tokens per vehicle through the frozen causal
// decoder, appending every layer's rotated keys and values to the KV cache
// that the tick reads. Its cost does not depend on the history length.
//
// Per call:  embed -> n_layers x [ RMSNorm+QKV (tcgen05 GEMM) -> rotary
//            embedding + cache-row writes -> causal attention over
//            [cached rows ; new rows] -> W_o + residual -> RMSNorm+gate/up+SiLU
//            -> W_d + residual ] -> residual stream out.
// The four projections reuse the tensor-core GEMM of the tick (gemm_tc.cu):
// norm gains folded into the packed weights, 1/rms applied in the epilogue from
// per-128-column sums of x^2, split K for the narrow residual GEMMs. The token
// count is n_new * B (4 for one vehicle), so the call streams every backbone
// weight once and is bound by HBM.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <thread>
#include <vector>

#include "../../include/fsx.h"
#include "device_util.cuh"
#include "gemm_tc.h"
#include "kernels.h"

namespace fsx {
void set_error_message(const char* msg);
}

namespace {

using fsx::kHeadDim;
constexpr int kMaxNew = 8;         // new tokens per vehicle and call
constexpr int kAttnWarps = 4;
constexpr int kRopePairs = kHeadDim / 2;

fsx_status fail(fsx_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  fsx::set_error_message(buf);
  return s;
}

#define FSX_CUDA(call)                                                                              \
  do {                                                                                              \
    cudaError_t e_ = (call);                                                                        \
    if (e_ != cudaSuccess) return fail(FSX_ERR_CUDA, "%s: %s (%s:%d)", #call, cudaGetErrorString(e_), \
                                       __FILE__, __LINE__);                                         \
  } while (0)

__device__ __forceinline__ int status_set(const int* status) {
  return *reinterpret_cast<const volatile int*>(status);
}

// ---- token rows in: x (fp32 residual stream), its fp16 copy and the per-token
// sums of x^2 over each 128-column group (the RMSNorm input of the QKV GEMM).
// Block 0 also checks the offsets and destination rows.
struct EmbedArgsA {
  const __nv_bfloat16* x_new;  // [M, d]
  const int64_t* offsets;      // [B + 1]
  const int64_t* dst;          // [B]
  int B, n_new, d;
  long long max_rows;
  float* x;
  __half* x16;
  float* ss;
  int ss_stride;
  int* status;
};

__global__ void __launch_bounds__(128) append_embed_kernel(const EmbedArgsA a) {
  const int m = blockIdx.x;
  if (m == 0 && threadIdx.x == 0) {
    const int64_t* off = a.offsets;
    bool ok = off[0] >= 0 && off[a.B] <= a.max_rows;
    for (int b = 0; b < a.B && ok; ++b) ok = off[b + 1] >= off[b];
    for (int b = 0; b < a.B && ok; ++b) {
      const int64_t lo = a.dst[b], hi = a.dst[b] + a.n_new;
      ok = lo >= 0 && hi <= a.max_rows && (hi <= off[0] || lo >= off[a.B]);
      for (int c = 0; c < b && ok; ++c) ok = hi <= a.dst[c] || lo >= a.dst[c] + a.n_new;
    }
    if (!ok) fsx::set_status(a.status, fsx::kStatusDeviceArg);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int g = warp; g < a.d / 128; g += 4) {
    const size_t idx = static_cast<size_t>(m) * a.d + g * 128 + lane * 4;
    const uint2 raw = *reinterpret_cast<const uint2*>(a.x_new + idx);
    const float v0 = __uint_as_float(raw.x << 16), v1 = __uint_as_float(raw.x & 0xffff0000u);
    const float v2 = __uint_as_float(raw.y << 16), v3 = __uint_as_float(raw.y & 0xffff0000u);
    *reinterpret_cast<float4*>(a.x + idx) = make_float4(v0, v1, v2, v3);
    *reinterpret_cast<uint2*>(a.x16 + idx) = make_uint2(fsx::pack_half2(v0, v1), fsx::pack_half2(v2, v3));
    const float ss = fsx::warp_sum(v0 * v0 + v1 * v1 + v2 * v2 + v3 * v3);
    if (lane == 0) a.ss[static_cast<size_t>(g) * a.ss_stride + m] = ss;
  }
}

// ---- rotary embedding of q and k at the new tokens' positions; k (rotated) and v
// written to the layer's cache rows dst[b] + i as bf16; q rotated in place.
struct RopeArgsA {
  __half* qkv;  // [M, 3 HD]: q | k | v
  int ld;
  int HD;
  const int64_t* offsets;
  const int64_t* dst;
  int n_new;
  double base;
  __nv_bfloat16* k_cache;  // this layer's rows
  __nv_bfloat16* v_cache;
  int* status;
};

__global__ void __launch_bounds__(kRopePairs) append_rope_kernel(const RopeArgsA r) {
  if (status_set(r.status)) return;
  const int m = blockIdx.x, h = blockIdx.y, j = threadIdx.x;  // pair (j, j + 64) of head h
  const int b = m / r.n_new, i = m - b * r.n_new;
  const long long pos = (r.offsets[b + 1] - r.offsets[b]) + i;
  const long long row = r.dst[b] + i;
  double sd, cd;
  sincos(static_cast<double>(pos) * pow(r.base, -2.0 * j / kHeadDim), &sd, &cd);
  const float s = static_cast<float>(sd), c = static_cast<float>(cd);
  __half* q = r.qkv + static_cast<size_t>(m) * r.ld + h * kHeadDim;
  const __half* k = q + r.HD;
  const __half* v = q + 2 * r.HD;
  const float q0 = __half2float(q[j]), q1 = __half2float(q[j + kRopePairs]);
  const float k0 = __half2float(k[j]), k1 = __half2float(k[j + kRopePairs]);
  q[j] = __float2half_rn(q0 * c - q1 * s);
  q[j + kRopePairs] = __float2half_rn(q0 * s + q1 * c);
  const size_t o = static_cast<size_t>(row) * r.HD + h * kHeadDim;
  r.k_cache[o + j] = __float2bfloat16_rn(k0 * c - k1 * s);
  r.k_cache[o + j + kRopePairs] = __float2bfloat16_rn(k0 * s + k1 * c);
  r.v_cache[o + j] = __float2bfloat16_rn(__half2float(v[j]));
  r.v_cache[o + j + kRopePairs] = __float2bfloat16_rn(__half2float(v[j + kRopePairs]));
}

// ---- causal attention of the new tokens of vehicle b, head h: keys are the
// vehicle's cached rows (positions 0 .. L_b-1) then its new rows (positions
// L_b ..); new token i sees every cached row and new rows 0 .. i. Warp w takes
// 32-key chunks w, w + 4, ...: lane l scores key 32c + l against every query
// (online softmax per query across the chunk), then owns value dims 4l..4l+3
// of the output. The four warps merge their states at the end.
struct AttnArgsA {
  const __half* qkv;  // rotated q at column h * 128 of row m
  int ld;
  int HD;
  const __nv_bfloat16* k_cache;
  const __nv_bfloat16* v_cache;
  const int64_t* offsets;
  const int64_t* dst;
  int n_new;
  __half* out;  // [M, HD]
  int* status;
};

__device__ __forceinline__ const __nv_bfloat16* key_row(const __nv_bfloat16* base, long long lo, long long L,
                                                        long long d0, int key, int HD, int h) {
  const long long row = key < L ? lo + key : d0 + (key - L);
  return base + static_cast<size_t>(row) * HD + h * kHeadDim;
}

__global__ void __launch_bounds__(kAttnWarps * 32) append_attn_kernel(const AttnArgsA a) {
  if (status_set(a.status)) return;
  __shared__ float qs[kMaxNew][kHeadDim];
  __shared__ float sm_m[kAttnWarps][kMaxNew], sm_l[kAttnWarps][kMaxNew];
  __shared__ float sm_o[kAttnWarps][kMaxNew][kHeadDim];
  const int b = blockIdx.x, h = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nq = a.n_new;
  const long long lo = a.offsets[b];
  const long long L = a.offsets[b + 1] - lo;
  const long long d0 = a.dst[b];
  const int N = static_cast<int>(L) + nq;
  const float scale = 1.4426950408889634f * rsqrtf(static_cast<float>(kHeadDim));  // log2(e) / sqrt(128)
  for (int t = threadIdx.x; t < nq * kHeadDim; t += blockDim.x) {
    const int qi = t / kHeadDim, dd = t - qi * kHeadDim;
    qs[qi][dd] = __half2float(a.qkv[static_cast<size_t>(b * nq + qi) * a.ld + h * kHeadDim + dd]) * scale;
  }
  __syncthreads();

  float m_run[kMaxNew], l_run[kMaxNew], o[kMaxNew][4];
#pragma unroll
  for (int qi = 0; qi < kMaxNew; ++qi) {
    m_run[qi] = -INFINITY;
    l_run[qi] = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e) o[qi][e] = 0.f;
  }
  for (int c0 = warp * 32; c0 < N; c0 += kAttnWarps * 32) {
    const int key = c0 + lane;
    float s[kMaxNew];
#pragma unroll
    for (int qi = 0; qi < kMaxNew; ++qi) s[qi] = 0.f;
    if (key < N) {
      const uint4* kr = reinterpret_cast<const uint4*>(key_row(a.k_cache, lo, L, d0, key, a.HD, h));
#pragma unroll 4
      for (int u = 0; u < kHeadDim / 8; ++u) {
        const uint4 raw = kr[u];
        float kv[8];
        kv[0] = __uint_as_float(raw.x << 16);
        kv[1] = __uint_as_float(raw.x & 0xffff0000u);
        kv[2] = __uint_as_float(raw.y << 16);
        kv[3] = __uint_as_float(raw.y & 0xffff0000u);
        kv[4] = __uint_as_float(raw.z << 16);
        kv[5] = __uint_as_float(raw.z & 0xffff0000u);
        kv[6] = __uint_as_float(raw.w << 16);
        kv[7] = __uint_as_float(raw.w & 0xffff0000u);
#pragma unroll
        for (int qi = 0; qi < kMaxNew; ++qi)
          if (qi < nq)
#pragma unroll
            for (int e = 0; e < 8; ++e) s[qi] = fmaf(qs[qi][u * 8 + e], kv[e], s[qi]);
      }
    }
    float p[kMaxNew];
#pragma unroll
    for (int qi = 0; qi < kMaxNew; ++qi) {
      // visible: a real key that is a cached row or a new row j <= qi
      const bool vis = qi < nq && key < N && (key < L || key - L <= qi);
      const float sv = vis ? s[qi] : -INFINITY;
      float mx = sv;
#pragma unroll
      for (int sh = 16; sh > 0; sh >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, sh));
      const float m_new = fmaxf(m_run[qi], mx);
      if (m_new == -INFINITY) {  // nothing visible yet for this query
        p[qi] = 0.f;
        continue;
      }
      const float alpha = exp2f(m_run[qi] - m_new);
      p[qi] = vis ? exp2f(sv - m_new) : 0.f;
      l_run[qi] = l_run[qi] * alpha + fsx::warp_sum(p[qi]);
      m_run[qi] = m_new;
#pragma unroll
      for (int e = 0; e < 4; ++e) o[qi][e] *= alpha;
    }
    const int n_chunk = min(32, N - c0);
    for (int kk = 0; kk < n_chunk; ++kk) {
      const uint2 raw = *reinterpret_cast<const uint2*>(key_row(a.v_cache, lo, L, d0, c0 + kk, a.HD, h) + lane * 4);
      const float v0 = __uint_as_float(raw.x << 16), v1 = __uint_as_float(raw.x & 0xffff0000u);
      const float v2 = __uint_as_float(raw.y << 16), v3 = __uint_as_float(raw.y & 0xffff0000u);
#pragma unroll
      for (int qi = 0; qi < kMaxNew; ++qi) {
        const float pk = __shfl_sync(0xffffffffu, p[qi], kk);
        o[qi][0] = fmaf(pk, v0, o[qi][0]);
        o[qi][1] = fmaf(pk, v1, o[qi][1]);
        o[qi][2] = fmaf(pk, v2, o[qi][2]);
        o[qi][3] = fmaf(pk, v3, o[qi][3]);
      }
    }
  }
#pragma unroll
  for (int qi = 0; qi < kMaxNew; ++qi) {
    if (lane == 0) {
      sm_m[warp][qi] = m_run[qi];
      sm_l[warp][qi] = l_run[qi];
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) sm_o[warp][qi][lane * 4 + e] = o[qi][e];
  }
  __syncthreads();
  for (int t = threadIdx.x; t < nq * kHeadDim; t += blockDim.x) {
    const int qi = t / kHeadDim, dd = t - qi * kHeadDim;
    float mm = -INFINITY;
#pragma unroll
    for (int w = 0; w < kAttnWarps; ++w) mm = fmaxf(mm, sm_m[w][qi]);
    float num = 0.f, den = 0.f;
#pragma unroll
    for (int w = 0; w < kAttnWarps; ++w) {
      const float f = sm_m[w][qi] == -INFINITY ? 0.f : exp2f(sm_m[w][qi] - mm);
      num += f * sm_o[w][qi][dd];
      den += f * sm_l[w][qi];
    }
    a.out[static_cast<size_t>(b * nq + qi) * a.HD + h * kHeadDim + dd] = __float2half_rn(den > 0.f ? num / den : 0.f);
  }
}

}  // namespace

struct fsx_append_s {
  fsx_append_config cfg{};
  int device = 0;
  bool concurrent = false;  // no kernel of a call waits on other CTAs (no split K)
  int sm_count = 0;
  int HD = 0;
  void* w_arena = nullptr;
  long long weight_bytes = 0;
  std::vector<const unsigned char*> w_qkv, w_o, w_gu, w_dn;
  CUtensorMap map_x16[3], map_o[3], map_h[3];
  float* x = nullptr;
  __half* x16 = nullptr;
  float* ss = nullptr;
  int ss_stride = 0;
  __half* qkv = nullptr;
  __half* o = nullptr;
  __half* hbuf = nullptr;
  float* gemm_part = nullptr;
  int* tile_count = nullptr;
  int* status = nullptr;
};

namespace {

void free_append(fsx_append_s* h) {
  if (!h) return;
  cudaSetDevice(h->device);
  cudaDeviceSynchronize();
  void* bufs[] = {h->w_arena, h->x, h->x16, h->ss, h->qkv, h->o, h->hbuf, h->gemm_part, h->tile_count, h->status};
  for (void* p : bufs)
    if (p) cudaFree(p);
  delete h;
}

fsx_status check_append_config(const fsx_append_config* c) {
  if (!c) return fail(FSX_ERR_INVALID_ARG, "config is NULL");
  if (c->n_layers <= 0 || c->d_model <= 0 || c->n_heads <= 0 || c->head_dim <= 0 || c->d_ff <= 0 ||
      c->n_new <= 0 || c->max_batch <= 0 || c->max_cache_rows < 0)
    return fail(FSX_ERR_INVALID_ARG, "config fields must be positive (max_cache_rows >= 0)");
  if (!(c->rope_base > 1.f)) return fail(FSX_ERR_INVALID_ARG, "rope_base must be > 1");
  if (c->head_dim != kHeadDim) return fail(FSX_ERR_UNSUPPORTED, "head_dim must be 128");
  if (c->d_model % 128 != 0) return fail(FSX_ERR_UNSUPPORTED, "d_model must be a multiple of 128");
  if (c->d_ff % 64 != 0) return fail(FSX_ERR_UNSUPPORTED, "d_ff must be a multiple of 64");
  if (c->n_new > kMaxNew) return fail(FSX_ERR_UNSUPPORTED, "n_new must be <= %d", kMaxNew);
  if (static_cast<long long>(c->n_new) * c->max_batch > 256)
    return fail(FSX_ERR_UNSUPPORTED, "n_new * max_batch must be <= 256");
  if (c->n_heads > 4096) return fail(FSX_ERR_UNSUPPORTED, "n_heads too large");
  return FSX_OK;
}

}  // namespace

extern "C" {

fsx_status fsx_append_create(const fsx_append_config* cfg, const fsx_append_weights* w, int device,
                             fsx_append_handle* out) {
  fsx::set_error_message("");
  if (!out) return fail(FSX_ERR_INVALID_ARG, "out handle pointer is NULL");
  *out = nullptr;
  fsx_status st = check_append_config(cfg);
  if (st != FSX_OK) return st;
  if (!w || !w->attn_norm || !w->wq || !w->wk || !w->wv || !w->wo || !w->mlp_norm || !w->w_gate || !w->w_up ||
      !w->w_down)
    return fail(FSX_ERR_INVALID_ARG, "a weight pointer is NULL");
  if (device < 0) return fail(FSX_ERR_INVALID_ARG, "device must be >= 0");
  int n_dev = 0;
  if (cudaGetDeviceCount(&n_dev) != cudaSuccess || n_dev == 0) return fail(FSX_ERR_CUDA, "no CUDA device available");
  if (device >= n_dev) return fail(FSX_ERR_INVALID_ARG, "device %d >= device count %d", device, n_dev);

  fsx_append_s* h = new fsx_append_s();
  h->cfg = *cfg;
  h->device = device;
  h->HD = cfg->n_heads * cfg->head_dim;
  const int L = cfg->n_layers, d = cfg->d_model, HD = h->HD, F = cfg->d_ff;
  auto bail = [&](fsx_status s) {
    free_append(h);
    return s;
  };
#define FSX_CUDA_H(call)                                                                                  \
  do {                                                                                                    \
    cudaError_t e_ = (call);                                                                              \
    if (e_ != cudaSuccess)                                                                                \
      return bail(fail(e_ == cudaErrorMemoryAllocation ? FSX_ERR_OOM : FSX_ERR_CUDA, "%s: %s", #call,    \
                       cudaGetErrorString(e_)));                                                          \
  } while (0)

  FSX_CUDA_H(cudaSetDevice(device));
  FSX_CUDA_H(cudaDeviceGetAttribute(&h->sm_count, cudaDevAttrMultiProcessorCount, device));
  FSX_CUDA_H(fsx::gemm_tc_set_attributes());

  // ---- weight tiles per layer [QKV | W_o | gate/up | W_d], 128-row x 64-K swizzled
  // images; RMSNorm gains folded into the K columns of QKV and gate/up; gate/up rows
  // interleaved so one 128-row tile holds gate rows 8j..8j+7 next to their up rows
  const size_t tile = fsx::kTcTileBytes;
  const size_t t_qkv = static_cast<size_t>(3 * HD / 128) * (d / 64), t_o = static_cast<size_t>(d / 128) * (HD / 64);
  const size_t t_gu = static_cast<size_t>(2 * F / 128) * (d / 64), t_dn = static_cast<size_t>(d / 128) * (F / 64);
  const size_t per_layer = (t_qkv + t_o + t_gu + t_dn) * tile;
  h->weight_bytes = static_cast<long long>(per_layer) * L;
  FSX_CUDA_H(cudaMalloc(&h->w_arena, per_layer * L));
  {
    std::vector<unsigned char> host(per_layer);
    const size_t hd_d = static_cast<size_t>(HD) * d;
    const int n_threads = std::max(1, std::min<int>(16, static_cast<int>(std::thread::hardware_concurrency())));
    // rows(r) -> source row r of the (row-permuted) matrix, N rows of K columns, optional per-K gain;
    // the n-tiles are spread over the threads
    auto pack_matrix = [&](auto rows, int N, int K, const float* gain, unsigned char* dst) {
      std::vector<std::thread> pool;
      for (int t = 0; t < n_threads; ++t)
        pool.emplace_back([&, t]() {
          const float* rp[128];
          for (int nt = t; nt < N / 128; nt += n_threads)
            for (int kt = 0; kt < K / 64; ++kt) {
              for (int r = 0; r < 128; ++r) rp[r] = rows(nt * 128 + r);
              fsx::pack_tc_tile(rp, gain, kt * 64,
                                reinterpret_cast<__half*>(dst + (static_cast<size_t>(nt) * (K / 64) + kt) * tile));
            }
        });
      for (auto& th : pool) th.join();
    };
    for (int l = 0; l < L; ++l) {
      unsigned char* base = host.data();
      const float* wq = w->wq + hd_d * l;
      const float* wk = w->wk + hd_d * l;
      const float* wv = w->wv + hd_d * l;
      pack_matrix(
          [&](int r) -> const float* {
            if (r < HD) return wq + static_cast<size_t>(r) * d;
            if (r < 2 * HD) return wk + static_cast<size_t>(r - HD) * d;
            return wv + static_cast<size_t>(r - 2 * HD) * d;
          },
          3 * HD, d, w->attn_norm + static_cast<size_t>(l) * d, base);
      const float* wo = w->wo + hd_d * l;
      pack_matrix([&](int r) -> const float* { return wo + static_cast<size_t>(r) * HD; }, d, HD, nullptr,
                  base + t_qkv * tile);
      const float* wg = w->w_gate + static_cast<size_t>(F) * d * l;
      const float* wu = w->w_up + static_cast<size_t>(F) * d * l;
      pack_matrix(
          [&](int q) -> const float* {
            const int blk = q >> 4, r = q & 15;
            return r < 8 ? wg + static_cast<size_t>(blk * 8 + r) * d : wu + static_cast<size_t>(blk * 8 + r - 8) * d;
          },
          2 * F, d, w->mlp_norm + static_cast<size_t>(l) * d, base + (t_qkv + t_o) * tile);
      const float* wd = w->w_down + static_cast<size_t>(d) * F * l;
      pack_matrix([&](int r) -> const float* { return wd + static_cast<size_t>(r) * F; }, d, F, nullptr,
                  base + (t_qkv + t_o + t_gu) * tile);
      FSX_CUDA_H(cudaMemcpy(static_cast<unsigned char*>(h->w_arena) + per_layer * l, host.data(), per_layer,
                            cudaMemcpyHostToDevice));
    }
  }
  for (int l = 0; l < L; ++l) {
    const unsigned char* base = static_cast<const unsigned char*>(h->w_arena) + per_layer * l;
    h->w_qkv.push_back(base);
    h->w_o.push_back(base + t_qkv * tile);
    h->w_gu.push_back(base + (t_qkv + t_o) * tile);
    h->w_dn.push_back(base + (t_qkv + t_o + t_gu) * tile);
  }

  // ---- workspace: token rows padded to whole 256-token tiles
  const size_t m_pad = (static_cast<size_t>(cfg->n_new) * cfg->max_batch + 255) / 256 * 256;
  FSX_CUDA_H(cudaMalloc(&h->x, m_pad * d * sizeof(float)));
  FSX_CUDA_H(cudaMalloc(&h->x16, m_pad * d * sizeof(__half)));
  h->ss_stride = static_cast<int>(m_pad);
  FSX_CUDA_H(cudaMalloc(&h->ss, static_cast<size_t>(d / 128) * m_pad * sizeof(float)));
  FSX_CUDA_H(cudaMalloc(&h->qkv, m_pad * 3 * HD * sizeof(__half)));
  FSX_CUDA_H(cudaMalloc(&h->o, m_pad * HD * sizeof(__half)));
  FSX_CUDA_H(cudaMalloc(&h->hbuf, m_pad * F * sizeof(__half)));
  FSX_CUDA_H(cudaMemset(h->x, 0, m_pad * d * sizeof(float)));
  FSX_CUDA_H(cudaMemset(h->x16, 0, m_pad * d * sizeof(__half)));
  FSX_CUDA_H(cudaMemset(h->ss, 0, static_cast<size_t>(d / 128) * m_pad * sizeof(float)));
  FSX_CUDA_H(cudaMemset(h->qkv, 0, m_pad * 3 * HD * sizeof(__half)));
  FSX_CUDA_H(cudaMemset(h->o, 0, m_pad * HD * sizeof(__half)));
  FSX_CUDA_H(cudaMemset(h->hbuf, 0, m_pad * F * sizeof(__half)));
  {
    const uint32_t boxes[3] = {48, 128, 256};  // index 0 (48-token tiles) is encoded but unused
    for (int i = 0; i < 3; ++i)
      if (!fsx::encode_act_map(&h->map_x16[i], h->x16, m_pad, d, boxes[i]) ||
          !fsx::encode_act_map(&h->map_o[i], h->o, m_pad, HD, boxes[i]) ||
          !fsx::encode_act_map(&h->map_h[i], h->hbuf, m_pad, F, boxes[i]))
        return bail(fail(FSX_ERR_CUDA, "tensor map encoding of the activation buffers failed"));
  }
  FSX_CUDA_H(cudaMalloc(&h->gemm_part, fsx::gemm_tc_part_bytes(h->sm_count)));
  FSX_CUDA_H(cudaMalloc(&h->tile_count, sizeof(int) * h->sm_count));
  FSX_CUDA_H(cudaMemset(h->tile_count, 0, sizeof(int) * h->sm_count));
  FSX_CUDA_H(cudaMalloc(&h->status, sizeof(int)));
  FSX_CUDA_H(cudaMemset(h->status, 0, sizeof(int)));
  FSX_CUDA_H(cudaDeviceSynchronize());
#undef FSX_CUDA_H
  *out = h;
  return FSX_OK;
}

fsx_status fsx_append_set_concurrent(fsx_append_handle h, int enable) {
  if (!h) return fail(FSX_ERR_INVALID_ARG, "handle is NULL");
  h->concurrent = enable != 0;
  return FSX_OK;
}

fsx_status fsx_append(fsx_append_handle h, void* const* k_cache, void* const* v_cache, const int64_t* d_offsets,
                      const int64_t* d_dst_rows, int B, const void* d_x_new, float* d_hidden, void* stream) {
  if (!h) return fail(FSX_ERR_INVALID_ARG, "handle is NULL");
  const fsx_append_config& c = h->cfg;
  if (!k_cache || !v_cache || !d_offsets || !d_dst_rows || !d_x_new || !d_hidden)
    return fail(FSX_ERR_INVALID_ARG, "a pointer argument is NULL");
  if (B < 1 || B > c.max_batch) return fail(FSX_ERR_INVALID_ARG, "B=%d outside 1..max_batch=%d", B, c.max_batch);
  for (int l = 0; l < c.n_layers; ++l)
    if (!k_cache[l] || !v_cache[l]) return fail(FSX_ERR_INVALID_ARG, "cache layer %d pointer is NULL", l);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  FSX_CUDA(cudaSetDevice(h->device));
  const int d = c.d_model, HD = h->HD, F = c.d_ff;
  const int M = B * c.n_new;
  // token tile of the GEMMs: 128 up to 128 tokens (an MMA of N = 128 costs the same as one of
  // N = 48 at one CTA per SM, and the weights bound the call), 256 above
  const int bn_i = M <= 128 ? 1 : 2;
  const int bn = bn_i == 1 ? 128 : 256;
  const int m_tiles = (M + bn - 1) / bn;

  EmbedArgsA ea{};
  ea.x_new = static_cast<const __nv_bfloat16*>(d_x_new);
  ea.offsets = d_offsets;
  ea.dst = d_dst_rows;
  ea.B = B;
  ea.n_new = c.n_new;
  ea.d = d;
  ea.max_rows = c.max_cache_rows;
  ea.x = h->x;
  ea.x16 = h->x16;
  ea.ss = h->ss;
  ea.ss_stride = h->ss_stride;
  ea.status = h->status;
  append_embed_kernel<<<M, 128, 0, st>>>(ea);
  FSX_CUDA(cudaGetLastError());

  for (int l = 0; l < c.n_layers; ++l) {
    fsx::TcGemmArgs g{};
    g.M = M;
    g.status = h->status;
    g.w = h->w_qkv[l];
    g.N = 3 * HD;
    g.K = d;
    g.y = h->qkv;
    g.ldy = 3 * HD;
    g.ss_in = h->ss;
    g.n_ss = d / 128;
    g.ss_stride = h->ss_stride;
    FSX_CUDA(fsx::launch_gemm_tc(h->map_x16[bn_i], g, bn, fsx::kEpiStore, true, st, false));

    RopeArgsA ra{};
    ra.qkv = h->qkv;
    ra.ld = 3 * HD;
    ra.HD = HD;
    ra.offsets = d_offsets;
    ra.dst = d_dst_rows;
    ra.n_new = c.n_new;
    ra.base = static_cast<double>(c.rope_base);
    ra.k_cache = static_cast<__nv_bfloat16*>(k_cache[l]);
    ra.v_cache = static_cast<__nv_bfloat16*>(v_cache[l]);
    ra.status = h->status;
    append_rope_kernel<<<dim3(M, c.n_heads), kRopePairs, 0, st>>>(ra);
    FSX_CUDA(cudaGetLastError());

    AttnArgsA aa{};
    aa.qkv = h->qkv;
    aa.ld = 3 * HD;
    aa.HD = HD;
    aa.k_cache = static_cast<const __nv_bfloat16*>(k_cache[l]);
    aa.v_cache = static_cast<const __nv_bfloat16*>(v_cache[l]);
    aa.offsets = d_offsets;
    aa.dst = d_dst_rows;
    aa.n_new = c.n_new;
    aa.out = h->o;
    aa.status = h->status;
    append_attn_kernel<<<dim3(B, c.n_heads), kAttnWarps * 32, 0, st>>>(aa);
    FSX_CUDA(cudaGetLastError());

    fsx::TcGemmArgs go{};
    go.M = M;
    go.status = h->status;
    go.w = h->w_o[l];
    go.N = d;
    go.K = HD;
    go.xo = h->x;
    go.xo16 = h->x16;
    go.ldxo = d;
    go.ss_out = h->ss;
    go.ss_stride = h->ss_stride;
    go.k_splits = h->concurrent ? 1 : fsx::gemm_tc_k_splits((d / 128) * m_tiles, HD / 64, h->sm_count);
    go.part = h->gemm_part;
    go.tile_count = h->tile_count;
    FSX_CUDA(fsx::launch_gemm_tc(h->map_o[bn_i], go, bn, fsx::kEpiResidual, false, st, false));

    fsx::TcGemmArgs gg{};
    gg.M = M;
    gg.status = h->status;
    gg.w = h->w_gu[l];
    gg.N = 2 * F;
    gg.K = d;
    gg.y = h->hbuf;
    gg.ldy = F;
    gg.ss_in = h->ss;
    gg.n_ss = d / 128;
    gg.ss_stride = h->ss_stride;
    FSX_CUDA(fsx::launch_gemm_tc(h->map_x16[bn_i], gg, bn, fsx::kEpiSwiglu, true, st, false));

    fsx::TcGemmArgs gd{};
    gd.M = M;
    gd.status = h->status;
    gd.w = h->w_dn[l];
    gd.N = d;
    gd.K = F;
    gd.xo = h->x;
    gd.xo16 = h->x16;
    gd.ldxo = d;
    gd.ss_out = h->ss;
    gd.ss_stride = h->ss_stride;
    gd.k_splits = h->concurrent ? 1 : fsx::gemm_tc_k_splits((d / 128) * m_tiles, F / 64, h->sm_count);
    gd.part = h->gemm_part;
    gd.tile_count = h->tile_count;
    FSX_CUDA(fsx::launch_gemm_tc(h->map_h[bn_i], gd, bn, fsx::kEpiResidual, false, st, false));
  }
  FSX_CUDA(cudaMemcpyAsync(d_hidden, h->x, static_cast<size_t>(M) * d * sizeof(float), cudaMemcpyDeviceToDevice, st));
  return FSX_OK;
}

fsx_status fsx_append_get_status(fsx_append_handle h, void* stream) {
  if (!h) return fail(FSX_ERR_INVALID_ARG, "handle is NULL");
  FSX_CUDA(cudaSetDevice(h->device));
  FSX_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  int v = 0;
  FSX_CUDA(cudaMemcpy(&v, h->status, sizeof(int), cudaMemcpyDeviceToHost));
  FSX_CUDA(cudaMemset(h->status, 0, sizeof(int)));
  return static_cast<fsx_status>(v);
}

long long fsx_append_weight_bytes(fsx_append_handle h) { return h ? h->weight_bytes : 0; }

void fsx_append_destroy(fsx_append_handle h) { free_append(h); }

}  // extern "C"
