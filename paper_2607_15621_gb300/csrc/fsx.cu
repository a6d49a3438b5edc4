// C ABI of the action-expert tick (include/fsx.h): handle creation with fp16
// weight packing, the per-tick launch sequence, CUDA-graph capture and replay,
// the device status word and the test/measurement entry points.
//
// Per tick (Sec. 3.1; the expert runs at every tick of Sec. 3.3 and reads the
// cache as-is):   embed -> 32 x [ RMSNorm+QKV -> Eq. 1 attention (+ merge)
//                 -> W_o + residual -> RMSNorm+gate/up+SiLU -> W_d + residual ]
//                 -> RMSNorm + waypoint head.
// Every launch uses programmatic dependent launch, so each kernel can fetch
// its weights while its predecessor finishes; the sequence for one batch size
// is captured once into a CUDA graph and replayed by every later tick.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <thread>
#include <vector>

#include "../../include/fsx.h"
#include "gemm_tc.h"
#include "kernels.h"
#include "persistent.h"
#include "tcgen05.cuh"

using fsx::TickArgs;

namespace {

thread_local char g_err[512] = "";

fsx_status fail(fsx_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

#define FSX_CUDA(call)                                                                              \
  do {                                                                                              \
    cudaError_t e_ = (call);                                                                        \
    if (e_ != cudaSuccess) return fail(FSX_ERR_CUDA, "%s: %s (%s:%d)", #call, cudaGetErrorString(e_), \
                                       __FILE__, __LINE__);                                         \
  } while (0)

constexpr int kClassQkv = 0, kClassAttn = 1, kClassWo = 2, kClassGateUp = 3, kClassDown = 4, kClassPersistent = 5;

}  // namespace

namespace fsx {
// Lets the other translation units of the library report a message through fsx_last_error().
void set_error_message(const char* msg) { snprintf(g_err, sizeof(g_err), "%s", msg ? msg : ""); }
}  // namespace fsx

struct fsx_handle_s {
  fsx_config cfg{};
  int device = 0;
  int sm_count = 0;
  int T = 0;
  int HD = 0;
  // packed fp16 weights
  void* w_arena = nullptr;
  long long weight_bytes = 0;
  std::vector<const unsigned char*> w_qkv, w_o, w_gu, w_dn;  // tcgen05 tile images per layer
  // 2-D tensor maps of the activation buffers for the token tile sizes 48 / 128 / 256
  CUtensorMap map_x16[4], map_o[4], map_h[4];  // token boxes of 48, 128, 256, 144 rows
  CUtensorMap map_w;                            // every packed weight tile (pair GEMM variant)
  bool pair_gemm = false;                       // QKV at 256-token tiles may run on CTA pairs (opt-in)
  // fp32 small parameters
  float* params = nullptr;
  float *act_emb = nullptr, *pos_emb = nullptr, *attn_norm = nullptr, *mlp_norm = nullptr;
  float *final_norm = nullptr, *head_w = nullptr, *head_b = nullptr;
  // workspace
  float* x = nullptr;
  __half* x16 = nullptr;
  float* ss = nullptr;   // per-row sums of x^2 over 128-column groups
  int ss_stride = 0;
  __half* qkv = nullptr;
  __half* o = nullptr;
  __half* hbuf = nullptr;
  float* part = nullptr;
  size_t part_bytes = 0;
  float* gemm_part = nullptr;   // split-K partial tiles of the residual GEMMs
  int* tile_count = nullptr;    // [sm_count] split arrivals per tile, zero between launches
  int* order = nullptr;         // [max_batch] vehicles by decreasing cache length (attention schedule)
  fsx::AttnPlan* plan = nullptr;  // [max_batch] the same schedule with each vehicle's cache range
  int* status = nullptr;
  TickArgs* d_args = nullptr;
  TickArgs h_args{};
  bool args_valid = false;
  // bf16 caches: TMA maps of every layer's K and V cache ([2 n_layers], device), re-encoded
  // whenever the cache pointers change; the tensor-core attention loads whole chunks with them
  CUtensorMap* d_cache_maps = nullptr;
  std::vector<CUtensorMap> h_cache_maps;
  // persistent single-vehicle tick
  bool persist_ok = false;
  void* p_arena = nullptr;
  long long p_layer_bytes = 0, p_a_cta = 0, p_b_offset = 0, p_b_cta = 0;
  float* p_x = nullptr;
  int* p_counters = nullptr;
  // host-buffer tick staging
  int64_t* st_offsets = nullptr;
  void* st_frames = nullptr;
  float* st_waypoints = nullptr;
  // graphs
  cudaStream_t cap_stream = nullptr;
  std::map<int, cudaGraphExec_t> graphs;
  std::map<int, cudaGraphExec_t> timed_graphs;
  bool timing = false;
  int timing_class = 0;
  std::vector<cudaEvent_t> tev;
  int timed_pairs = 0;
  bool timed_pending = false;
  cudaEvent_t last_tick = nullptr;
  cudaStream_t last_stream = nullptr;
  bool has_last = false;
  std::mutex mu;
  unsigned long long wait_limit_ns = 1000000000ull;  // device-wide counter waits of the single-launch tick
  // the ten-token layout (paper_tokens.cu): two-layer head and state MLP parameters,
  // assembled frame rows; null for the 42-token tick
  float* paper_params = nullptr;
  const float* paper_head = nullptr;
  const float* paper_state_w = nullptr;
  float* paper_frames = nullptr;
  int paper_visual_dtype = 0;
};

namespace {

int attention_splits(const fsx_handle_s* h, int B) {
  const int work = B * h->cfg.n_heads;
  int s = (2 * h->sm_count) / std::max(work, 1);
  return std::min(std::max(s, 1), 8);  // <= 8: the splits merge inside one thread-block cluster
}

fsx_status check_config(const fsx_config* c) {
  if (!c) return fail(FSX_ERR_INVALID_ARG, "config is NULL");
  if (c->n_layers <= 0 || c->d_model <= 0 || c->n_heads <= 0 || c->head_dim <= 0 || c->d_ff <= 0 ||
      c->n_action <= 0 || c->n_frame < 0 || c->n_waypoints <= 0 || c->max_batch <= 0 ||
      c->max_total_cache_tokens < 0)
    return fail(FSX_ERR_INVALID_ARG, "config fields must be positive (n_frame, max_total_cache_tokens >= 0)");
  if ((c->cache_dtype != FSX_F32 && c->cache_dtype != FSX_BF16) ||
      (c->frame_dtype != FSX_F32 && c->frame_dtype != FSX_BF16))
    return fail(FSX_ERR_INVALID_ARG, "cache_dtype / frame_dtype must be FSX_F32 or FSX_BF16");
  const int T = c->n_action + c->n_frame;
  if (c->n_waypoints > T) return fail(FSX_ERR_INVALID_ARG, "n_waypoints exceeds the token count");
  if (c->head_dim != fsx::kHeadDim) return fail(FSX_ERR_UNSUPPORTED, "head_dim must be 128");
  if (c->d_model % 128 != 0 || c->d_model > 1024) return fail(FSX_ERR_UNSUPPORTED, "d_model must be a multiple of 128, <= 1024");
  if (c->d_ff % 64 != 0) return fail(FSX_ERR_UNSUPPORTED, "d_ff must be a multiple of 64");
  if (T > fsx::kTokTile) return fail(FSX_ERR_UNSUPPORTED, "n_action + n_frame must be <= 48");
  if (c->n_layers > fsx::kMaxLayers) return fail(FSX_ERR_UNSUPPORTED, "n_layers must be <= 128");
  if (c->n_heads > 4096) return fail(FSX_ERR_UNSUPPORTED, "n_heads too large");
  return FSX_OK;
}

// fp32 rows -> fp16 swizzled K-major operand images of the tensor core, one
// rows x 128-byte image per 64-wide K slice (optional per-K gain folded in)
template <typename RowFn>
void pack_sw128(RowFn row, int rows, int K, const float* gain, unsigned char* out) {
  for (int r = 0; r < rows; ++r) {
    const float* src = row(r);
    for (int k = 0; k < K; ++k)
      *reinterpret_cast<__half*>(out + fsx::sw128_offset(rows, r, k)) =
          __float2half_rn(src[k] * (gain ? gain[k] : 1.f));
  }
}

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

bool use_persistent(const fsx_handle_s* h, int B) {
  if (B != 1 || !h->persist_ok) return false;
  const char* off = std::getenv("FSX_DISABLE_PERSISTENT");
  return !(off && off[0] == '1');
}

fsx_status enqueue_tick(fsx_handle_s* h, int B, cudaStream_t st, __half* attn_capture, bool timed) {
  const fsx_config& c = h->cfg;
  const int d = c.d_model, HD = h->HD, F = c.d_ff, T = h->T;
  const int M = B * T;
  const bool pdl = true;
  int pair = 0;
  auto mark = [&](int cls, bool begin) -> cudaError_t {
    if (!timed || cls != h->timing_class) return cudaSuccess;
    cudaEvent_t ev = h->tev[2 * pair + (begin ? 0 : 1)];
    if (!begin) ++pair;
    return cudaEventRecordWithFlags(ev, st, cudaEventRecordExternal);
  };

  if (use_persistent(h, B)) {
    fsx::PersistArgs pa{};
    pa.warena = static_cast<const unsigned char*>(h->p_arena);
    pa.layer_bytes = h->p_layer_bytes;
    pa.a_cta_bytes = h->p_a_cta;
    pa.b_offset = h->p_b_offset;
    pa.b_cta_bytes = h->p_b_cta;
    pa.act_emb = h->act_emb;
    pa.pos_emb = h->pos_emb;
    pa.final_norm = h->final_norm;
    pa.head_w = h->head_w;
    pa.head_b = h->head_b;
    pa.targs = h->d_args;
    pa.n_layers = c.n_layers;
    pa.d = d;
    pa.H = c.n_heads;
    pa.F = F;
    pa.n_action = c.n_action;
    pa.n_frame = c.n_frame;
    pa.n_waypoints = c.n_waypoints;
    pa.n_b_clusters = F / 64;
    pa.frame_dtype = c.frame_dtype;
    pa.max_total = c.max_total_cache_tokens;
    pa.X = h->p_x;
    pa.counters = h->p_counters;
    pa.status = h->status;
    pa.attn_capture = attn_capture;
    pa.head = h->paper_head == nullptr ? 1 : 0;
    pa.wait_limit_ns = h->wait_limit_ns;
    FSX_CUDA(cudaMemsetAsync(h->p_counters, 0, sizeof(int) * (2 * c.n_layers + 1), st));
    FSX_CUDA(mark(kClassPersistent, true));
    FSX_CUDA(fsx::launch_persistent(pa, c.cache_dtype, st));
    FSX_CUDA(mark(kClassPersistent, false));
    if (h->paper_head != nullptr) {  // the two-layer head over the final residual buffer
      fsx::Head2Args h2{};
      h2.x = h->p_x + static_cast<size_t>((2 * c.n_layers) % 3) * fsx::kTokTile * d;
      h2.vehicle_rows = 0;
      h2.final_norm = h->final_norm;
      h2.w = h->paper_head;
      h2.targs = h->d_args;
      h2.d = d;
      h2.n_waypoints = c.n_waypoints;
      h2.B = 1;
      h2.status = h->status;
      FSX_CUDA(fsx::launch_head2(h2, st, false));
    }
    if (timed) h->timed_pairs = pair;
    return FSX_OK;
  }

  fsx::EmbedArgs ea{};
  ea.act_emb = h->act_emb;
  ea.pos_emb = h->pos_emb;
  ea.targs = h->d_args;
  ea.frame_dtype = c.frame_dtype;
  ea.n_action = c.n_action;
  ea.n_frame = c.n_frame;
  ea.d = d;
  ea.B = B;
  ea.max_total = c.max_total_cache_tokens;
  ea.x = h->x;
  ea.x16 = h->x16;
  ea.ss = h->ss;
  ea.ss_stride = h->ss_stride;
  ea.order = h->order;
  ea.plan = h->plan;
  ea.status = h->status;
  FSX_CUDA(fsx::launch_embed(ea, st, pdl));

  // 48-row QKV tiles: 256 CTAs at two per SM run as one wave
  // token tile of the tensor-core GEMMs: 48 for one vehicle, then 128 / 256
  const int bn_i = M <= 48 ? 0 : (M <= 1024 ? 1 : 2);
  const int bn = bn_i == 0 ? 48 : (bn_i == 1 ? 128 : 256);
  // QKV (N = 12288) has tiles to spare: 256-token tiles halve its MMA instructions (one
  // tcgen05.mma costs the same for any N up to 256) whenever M exceeds one 48-token tile
  const int bq_i = M <= 48 ? 0 : 2;
  const int bq = bq_i == 0 ? 48 : 256;
  // The residual GEMMs (N = d) have only d / 128 weight tiles: with 256-token tiles they
  // fill about half the SMs. 144-token tiles give one tile per SM up to 38 x 144 tokens.
  const int rtiles144 = (d / 128) * ((M + 143) / 144);
  const int rbn_i = (bn_i == 2 && rtiles144 <= h->sm_count) ? 3 : bn_i;
  const int rbn = rbn_i == 3 ? 144 : bn;
  // QKV on CTA pairs (M = 256 tcgen05.mma.cta_group::2, half the token rows staged per SM)
  // when opted in, from 2048 tokens on. With the TMA-store epilogue the single-CTA kernel is
  // the faster one (5376 tokens: 60.7 against 67.3 us per launch), so it is the default.
  const bool qkv_pair = h->pair_gemm && bq == 256 && M >= 2048;
  const int S = attention_splits(h, B);

  for (int l = 0; l < c.n_layers; ++l) {
    fsx::TcGemmArgs g{};
    g.M = M;
    g.status = h->status;
    // RMSNorm + [W_q; W_k; W_v] (norm gain folded into the tiles)
    g.w = h->w_qkv[l];
    g.N = 3 * HD;
    g.K = d;
    g.y = h->qkv;
    g.ldy = 3 * HD;
    g.ss_in = h->ss;
    g.n_ss = d / 128;
    g.ss_stride = h->ss_stride;
    FSX_CUDA(mark(kClassQkv, true));
    g.w_tile0 = static_cast<int>((g.w - static_cast<const unsigned char*>(h->w_arena)) / fsx::kTcTileBytes);
    if (qkv_pair)
      FSX_CUDA(fsx::launch_gemm_tc(h->map_x16[1], g, bq, fsx::kEpiStore, true, st, pdl, &h->map_w));
    else
      FSX_CUDA(fsx::launch_gemm_tc(h->map_x16[bq_i], g, bq, fsx::kEpiStore, true, st, pdl));
    FSX_CUDA(mark(kClassQkv, false));

    // Eq. 1 over [cache_l ; own]
    fsx::AttnArgs a{};
    a.q = h->qkv;
    a.q_stride = 3 * HD;
    a.k_own = h->qkv + HD;
    a.v_own = h->qkv + 2 * HD;
    a.own_stride = 3 * HD;
    a.n_q = T;
    a.n_own = T;
    a.targs = h->d_args;
    a.layer = l;
    a.max_total = c.max_total_cache_tokens;
    a.n_heads = c.n_heads;
    a.n_splits = S;
    a.out = h->o;
    a.out_stride = HD;
    a.lse = nullptr;
    a.part_o = h->part;
    a.part_lse = h->part + static_cast<size_t>(B) * c.n_heads * S * fsx::kTokTile * fsx::kHeadDim;
    a.order = h->order;
    a.plan = h->plan;
    a.cache_maps = h->d_cache_maps;
    a.status = h->status;
    FSX_CUDA(mark(kClassAttn, true));
    FSX_CUDA(fsx::launch_attention(a, B, c.cache_dtype, st, pdl));
    FSX_CUDA(mark(kClassAttn, false));
    if (attn_capture) {
      FSX_CUDA(cudaMemcpyAsync(attn_capture + static_cast<size_t>(l) * M * HD, h->o,
                               static_cast<size_t>(M) * HD * sizeof(__half), cudaMemcpyDeviceToDevice, st));
    }

    // x += o W_o^T
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
    go.k_splits = fsx::gemm_tc_k_splits((d / 128) * ((M + rbn - 1) / rbn), HD / 64, h->sm_count);
    go.part = h->gemm_part;
    go.tile_count = h->tile_count;
    FSX_CUDA(mark(kClassWo, true));
    FSX_CUDA(fsx::launch_gemm_tc(h->map_o[rbn_i], go, rbn, fsx::kEpiResidual, false, st, pdl));
    FSX_CUDA(mark(kClassWo, false));

    // h = silu(RMSNorm(x) W_g^T) * (RMSNorm(x) W_u^T)
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
    FSX_CUDA(mark(kClassGateUp, true));
    FSX_CUDA(fsx::launch_gemm_tc(h->map_x16[bn_i], gg, bn, fsx::kEpiSwiglu, true, st, pdl));
    FSX_CUDA(mark(kClassGateUp, false));

    // x += h W_d^T
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
    gd.k_splits = fsx::gemm_tc_k_splits((d / 128) * ((M + rbn - 1) / rbn), F / 64, h->sm_count);
    gd.part = h->gemm_part;
    gd.tile_count = h->tile_count;
    FSX_CUDA(mark(kClassDown, true));
    FSX_CUDA(fsx::launch_gemm_tc(h->map_h[rbn_i], gd, rbn, fsx::kEpiResidual, false, st, pdl));
    FSX_CUDA(mark(kClassDown, false));
  }

  fsx::HeadArgs ha{};
  ha.x = h->x;
  ha.final_norm = h->final_norm;
  ha.head_w = h->head_w;
  ha.head_b = h->head_b;
  ha.targs = h->d_args;
  ha.out = nullptr;
  ha.d = d;
  ha.T = T;
  ha.n_waypoints = c.n_waypoints;
  ha.B = B;
  ha.status = h->status;
  if (h->paper_head != nullptr) {
    fsx::Head2Args h2{};
    h2.x = h->x;
    h2.vehicle_rows = T;
    h2.final_norm = h->final_norm;
    h2.w = h->paper_head;
    h2.targs = h->d_args;
    h2.d = d;
    h2.n_waypoints = c.n_waypoints;
    h2.B = B;
    h2.status = h->status;
    FSX_CUDA(fsx::launch_head2(h2, st, pdl));
  } else {
    FSX_CUDA(fsx::launch_head(ha, st, pdl));
  }
  if (timed) h->timed_pairs = pair;
  return FSX_OK;
}

fsx_status get_graph(fsx_handle_s* h, int B, bool timed, cudaGraphExec_t* out) {
  auto& map = timed ? h->timed_graphs : h->graphs;
  auto it = map.find(B);
  if (it != map.end()) {
    *out = it->second;
    return FSX_OK;
  }
  FSX_CUDA(cudaStreamBeginCapture(h->cap_stream, cudaStreamCaptureModeThreadLocal));
  fsx_status s = enqueue_tick(h, B, h->cap_stream, nullptr, timed);
  cudaGraph_t graph = nullptr;
  cudaError_t e = cudaStreamEndCapture(h->cap_stream, &graph);
  if (s != FSX_OK) {
    if (graph) cudaGraphDestroy(graph);
    return s;
  }
  if (e != cudaSuccess) return fail(FSX_ERR_CUDA, "graph capture failed: %s", cudaGetErrorString(e));
  cudaGraphExec_t exec = nullptr;
  e = cudaGraphInstantiate(&exec, graph, 0);
  cudaGraphDestroy(graph);
  if (e != cudaSuccess) return fail(FSX_ERR_CUDA, "graph instantiate failed: %s", cudaGetErrorString(e));
  map[B] = exec;
  *out = exec;
  return FSX_OK;
}

fsx_status check_tick_args(fsx_handle_s* h, const void* const* k_cache, const void* const* v_cache,
                           const void* offsets, int B, const void* frames, const void* waypoints) {
  if (!h) return fail(FSX_ERR_INVALID_ARG, "handle is NULL");
  if (B < 1 || B > h->cfg.max_batch) return fail(FSX_ERR_INVALID_ARG, "B=%d outside 1..max_batch=%d", B, h->cfg.max_batch);
  if (!k_cache || !v_cache) return fail(FSX_ERR_INVALID_ARG, "k_cache / v_cache pointer arrays are NULL");
  if (!offsets) return fail(FSX_ERR_INVALID_ARG, "offsets is NULL");
  if (!frames) return fail(FSX_ERR_INVALID_ARG, "frames is NULL");
  if (!waypoints) return fail(FSX_ERR_INVALID_ARG, "waypoints is NULL");
  return FSX_OK;
}

// Upload the per-tick pointers when they changed and order this tick after the
// previous one if it was issued on another stream.
fsx_status prepare_tick(fsx_handle_s* h, const void* const* k_cache, const void* const* v_cache,
                        const int64_t* d_offsets, const int64_t* d_starts, const void* d_frames, float* d_waypoints,
                        cudaStream_t st) {
  FSX_CUDA(cudaSetDevice(h->device));
  if (h->has_last && h->last_stream != st) FSX_CUDA(cudaStreamWaitEvent(st, h->last_tick, 0));
  TickArgs a{};
  for (int l = 0; l < h->cfg.n_layers; ++l) {
    a.k_cache[l] = k_cache[l];
    a.v_cache[l] = v_cache[l];
  }
  a.offsets = d_offsets;
  a.starts = d_starts;
  a.frames = d_frames;
  a.waypoints = d_waypoints;
  if (!h->args_valid || std::memcmp(&a, &h->h_args, sizeof(TickArgs)) != 0) {
    const bool caches_changed = !h->args_valid || std::memcmp(a.k_cache, h->h_args.k_cache, sizeof(a.k_cache)) != 0 ||
                                std::memcmp(a.v_cache, h->h_args.v_cache, sizeof(a.v_cache)) != 0;
    h->h_args = a;
    FSX_CUDA(cudaMemcpyAsync(h->d_args, &h->h_args, sizeof(TickArgs), cudaMemcpyHostToDevice, st));
    if (caches_changed && h->d_cache_maps != nullptr) {
      // the map of a NULL pointer stays zero: a layer without cache rows never loads through it
      std::memset(h->h_cache_maps.data(), 0, h->h_cache_maps.size() * sizeof(CUtensorMap));
      for (int l = 0; l < h->cfg.n_layers; ++l)
        for (int t = 0; t < 2; ++t) {
          const void* base = t == 0 ? a.k_cache[l] : a.v_cache[l];
          if (base != nullptr &&
              !fsx::encode_cache_map(&h->h_cache_maps[2 * l + t], base,
                                     static_cast<uint64_t>(h->cfg.max_total_cache_tokens), h->cfg.n_heads))
            return fail(FSX_ERR_INVALID_ARG, "a cache pointer is not 16-byte aligned (tensor map encoding failed)");
        }
      FSX_CUDA(cudaMemcpyAsync(h->d_cache_maps, h->h_cache_maps.data(), h->h_cache_maps.size() * sizeof(CUtensorMap),
                               cudaMemcpyHostToDevice, st));
    }
    h->args_valid = true;
  }
  return FSX_OK;
}

fsx_status finish_tick(fsx_handle_s* h, cudaStream_t st) {
  FSX_CUDA(cudaEventRecord(h->last_tick, st));
  h->last_stream = st;
  h->has_last = true;
  return FSX_OK;
}

void free_handle(fsx_handle_s* h) {
  if (!h) return;
  cudaSetDevice(h->device);
  cudaDeviceSynchronize();
  for (auto& kv : h->graphs) cudaGraphExecDestroy(kv.second);
  for (auto& kv : h->timed_graphs) cudaGraphExecDestroy(kv.second);
  for (cudaEvent_t e : h->tev) cudaEventDestroy(e);
  if (h->last_tick) cudaEventDestroy(h->last_tick);
  if (h->cap_stream) cudaStreamDestroy(h->cap_stream);
  if (h->paper_params) cudaFree(h->paper_params);
  if (h->paper_frames) cudaFree(h->paper_frames);
  void* bufs[] = {h->p_arena, h->p_x, h->p_counters, h->w_arena, h->params, h->x, h->x16, h->ss, h->qkv, h->o, h->hbuf, h->part,
                  h->gemm_part, h->tile_count, h->order, h->plan, h->status, h->d_args, h->d_cache_maps,
                  h->st_offsets, h->st_frames, h->st_waypoints};
  for (void* p : bufs)
    if (p) cudaFree(p);
  delete h;
}

}  // namespace

namespace fsx {

// hooks of the ten-token layout (paper_tokens.cu)
fsx_status paper_attach(fsx_handle h, float* d_params, const float* d_head, float* d_frames, const float* d_state_w,
                        int visual_dtype) {
  h->paper_params = d_params;
  h->paper_head = d_head;
  h->paper_frames = d_frames;
  h->paper_state_w = d_state_w;
  h->paper_visual_dtype = visual_dtype;
  return FSX_OK;
}
float* paper_frames(fsx_handle h) { return h->paper_frames; }
const float* paper_state_weights(fsx_handle h) { return h->paper_state_w; }
int paper_device(fsx_handle h) { return h->device; }
int paper_max_batch(fsx_handle h) { return h->cfg.max_batch; }
int paper_d(fsx_handle h) { return h->cfg.d_model; }
int paper_visual_dtype(fsx_handle h) { return h->paper_visual_dtype; }
// order work on `st` after the handle's previous tick when that ran on another stream
cudaError_t paper_order_after_last_tick(fsx_handle h, cudaStream_t st) {
  std::lock_guard<std::mutex> lock(h->mu);
  if (h->has_last && h->last_stream != st) return cudaStreamWaitEvent(st, h->last_tick, 0);
  return cudaSuccess;
}

}  // namespace fsx

extern "C" {

const char* fsx_last_error(void) { return g_err; }

fsx_status fsx_create(const fsx_config* cfg, const fsx_weights* w, int device, fsx_handle* out) {
  g_err[0] = '\0';
  if (!out) return fail(FSX_ERR_INVALID_ARG, "out handle pointer is NULL");
  *out = nullptr;
  fsx_status s = check_config(cfg);
  if (s != FSX_OK) return s;
  if (!w || !w->act_emb || !w->pos_emb || !w->attn_norm || !w->wq || !w->wk || !w->wv || !w->wo ||
      !w->mlp_norm || !w->w_gate || !w->w_up || !w->w_down || !w->final_norm || !w->head_w || !w->head_b)
    return fail(FSX_ERR_INVALID_ARG, "a weight pointer is NULL");
  if (device < 0) return fail(FSX_ERR_INVALID_ARG, "device must be >= 0");
  const char* fa = std::getenv("FSX_TEST_FAIL_ALLOC");
  if (fa && fa[0] == '1') return fail(FSX_ERR_OOM, "allocation failure forced by FSX_TEST_FAIL_ALLOC");

  int n_dev = 0;
  if (cudaGetDeviceCount(&n_dev) != cudaSuccess || n_dev == 0) return fail(FSX_ERR_CUDA, "no CUDA device available");
  if (device >= n_dev) return fail(FSX_ERR_INVALID_ARG, "device %d >= device count %d", device, n_dev);

  fsx_handle_s* h = new fsx_handle_s();
  h->cfg = *cfg;
  h->device = device;
  h->T = cfg->n_action + cfg->n_frame;
  h->HD = cfg->n_heads * cfg->head_dim;
  const int L = cfg->n_layers, d = cfg->d_model, HD = h->HD, F = cfg->d_ff, T = h->T;

  auto bail = [&](fsx_status st) {
    free_handle(h);
    return st;
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
  FSX_CUDA_H(fsx::attention_set_attributes());

  // ---- tcgen05 weight tiles: per layer [QKV | W_o | gate/up | W_d], each matrix as
  // 128-row x 64-K tiles in the swizzled shared-memory image (n-tile major)
  const size_t tile = fsx::kTcTileBytes;
  const size_t t_qkv = static_cast<size_t>(3 * HD / 128) * (d / 64), t_o = static_cast<size_t>(d / 128) * (HD / 64);
  const size_t t_gu = static_cast<size_t>(2 * F / 128) * (d / 64), t_dn = static_cast<size_t>(d / 128) * (F / 64);
  const size_t per_layer = (t_qkv + t_o + t_gu + t_dn) * tile;
  const size_t arena = per_layer * L;
  h->weight_bytes = static_cast<long long>(arena);
  FSX_CUDA_H(cudaMalloc(&h->w_arena, arena));
  {
    std::vector<__half> host(arena / 2);
    const size_t hd_d = static_cast<size_t>(HD) * d;
    // rows(r) -> source row r of the (row-permuted) matrix; K columns; optional per-K gain
    auto pack_matrix = [&](auto rows, int N, int K, const float* gain, unsigned char* out) {
      const float* rp[128];
      for (int nt = 0; nt < N / 128; ++nt)
        for (int kt = 0; kt < K / 64; ++kt) {
          for (int r = 0; r < 128; ++r) rp[r] = rows(nt * 128 + r);
          fsx::pack_tc_tile(rp, gain, kt * 64,
                            reinterpret_cast<__half*>(out + (static_cast<size_t>(nt) * (K / 64) + kt) * tile));
        }
    };
    auto pack_layer = [&](int l) {
      unsigned char* base = reinterpret_cast<unsigned char*>(host.data()) + per_layer * l;
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
      // packed row p: block p/16, rows 0..7 gate rows 8*(p/16)+r, rows 8..15 the matching up rows
      pack_matrix(
          [&](int q) -> const float* {
            const int blk = q >> 4, r = q & 15;
            return r < 8 ? wg + static_cast<size_t>(blk * 8 + r) * d : wu + static_cast<size_t>(blk * 8 + r - 8) * d;
          },
          2 * F, d, w->mlp_norm + static_cast<size_t>(l) * d, base + (t_qkv + t_o) * tile);
      const float* wd = w->w_down + static_cast<size_t>(d) * F * l;
      pack_matrix([&](int r) -> const float* { return wd + static_cast<size_t>(r) * F; }, d, F, nullptr,
                  base + (t_qkv + t_o + t_gu) * tile);
    };
    const int n_threads = std::max(1, std::min<int>(16, static_cast<int>(std::thread::hardware_concurrency())));
    std::vector<std::thread> pool;
    for (int t = 0; t < n_threads; ++t)
      pool.emplace_back([&, t]() {
        for (int l = t; l < L; l += n_threads) pack_layer(l);
      });
    for (auto& th : pool) th.join();
    FSX_CUDA_H(cudaMemcpy(h->w_arena, host.data(), arena, cudaMemcpyHostToDevice));
  }
  // the pair GEMM variant (CTA pairs on tcgen05.mma.cta_group::2, opted into by
  // FSX_PAIR_GEMM=1 at handle creation) loads the weight tiles through one map over the arena
  const char* pair_env = std::getenv("FSX_PAIR_GEMM");
  h->pair_gemm = fsx::gemm_tc_pair_clusters() > 0 && pair_env != nullptr && std::strcmp(pair_env, "1") == 0 &&
                 arena / tile <= 0x7fffffffull && fsx::encode_weight_map(&h->map_w, h->w_arena, arena / tile);
  for (int l = 0; l < L; ++l) {
    const unsigned char* base = static_cast<const unsigned char*>(h->w_arena) + per_layer * l;
    h->w_qkv.push_back(base);
    h->w_o.push_back(base + t_qkv * tile);
    h->w_gu.push_back(base + (t_qkv + t_o) * tile);
    h->w_dn.push_back(base + (t_qkv + t_o + t_gu) * tile);
  }

  // ---- stream-ordered weights of the persistent single-vehicle tick
  {
    const int H = cfg->n_heads;
    const int n_b = F / 64;
    int max_clusters = 0;
    const bool shape_ok = d == 512 && T <= fsx::kTokTile && F % 64 == 0 && n_b <= H &&
                          H * fsx::kPersistCluster <= h->sm_count && std::getenv("FSX_NO_PERSISTENT_BUILD") == nullptr;
    if (shape_ok && fsx::persistent_set_attributes(d) == cudaSuccess)
      max_clusters = fsx::persistent_max_clusters(d, cfg->cache_dtype);
    cudaGetLastError();
    if (shape_ok && max_clusters >= H) {
      const int G = H * fsx::kPersistCluster;
      const long long chunk = fsx::kPersistChunk;
      h->p_a_cta = chunk * fsx::kPersistAChunks;
      h->p_b_cta = chunk * fsx::kPersistBChunks;
      h->p_b_offset = h->p_a_cta * G;
      h->p_layer_bytes = h->p_b_offset + h->p_b_cta * n_b * fsx::kPersistCluster;
      const size_t total = static_cast<size_t>(h->p_layer_bytes) * L;
      FSX_CUDA_H(cudaMalloc(&h->p_arena, total));
      std::vector<__half> host(total / 2);
      const size_t hd_d = static_cast<size_t>(HD) * d;
      auto pack_layer = [&](int l) {
        unsigned char* base = reinterpret_cast<unsigned char*>(host.data()) + static_cast<size_t>(h->p_layer_bytes) * l;
        const float* g1 = w->attn_norm + static_cast<size_t>(l) * d;
        const float* g2 = w->mlp_norm + static_cast<size_t>(l) * d;
        for (int cta = 0; cta < G; ++cta) {
          const int head = cta / fsx::kPersistCluster, rank = cta % fsx::kPersistCluster;
          unsigned char* a = base + static_cast<size_t>(cta) * h->p_a_cta;
          const float* mats[3] = {w->wq + hd_d * l, w->wk + hd_d * l, w->wv + hd_d * l};
          // rows 32j..32j+31: dims 32 rank .. 32 rank + 31 of head h in W_q, W_k, W_v
          pack_sw128([&](int r) -> const float* {
            return mats[r / 32] + static_cast<size_t>(head * fsx::kHeadDim + rank * 32 + r % 32) * d;
          }, 96, d, g1, a);
          // 128 output columns of this rank x this head's 128 inputs
          const float* wo = w->wo + hd_d * l;
          pack_sw128([&](int r) -> const float* {
            return wo + static_cast<size_t>(rank * 128 + r) * HD + head * fsx::kHeadDim;
          }, 128, fsx::kHeadDim, nullptr, a + 96 * 128 * (d / 64));  // after the 96-row QKV images
        }
        const float* wg = w->w_gate + static_cast<size_t>(F) * d * l;
        const float* wu = w->w_up + static_cast<size_t>(F) * d * l;
        const float* wd = w->w_down + static_cast<size_t>(d) * F * l;
        for (int cta = 0; cta < n_b * fsx::kPersistCluster; ++cta) {
          const int cl = cta / fsx::kPersistCluster, rank = cta % fsx::kPersistCluster;
          unsigned char* b = base + h->p_b_offset + static_cast<size_t>(cta) * h->p_b_cta;
          // the cluster's 128 gate/up rows over this rank's K quarter (columns 128 rank ..):
          // rows 32s + i, i < 16: gate column 64 cl + 16 s + i; i >= 16: the matching up column
          pack_sw128([&](int r) -> const float* {
            const int s_ = r / 32, i = r % 32;
            const int col = cl * 64 + s_ * 16 + i % 16;
            return (i < 16 ? wg : wu) + static_cast<size_t>(col) * d + rank * 128;
          }, 128, 128, g2 + rank * 128, b);
          // 128 output columns x this cluster's 64 SwiGLU inputs
          pack_sw128([&](int r) -> const float* {
            return wd + static_cast<size_t>(rank * 128 + r) * F + cl * 64;
          }, 128, 64, nullptr, b + 128 * 128 * 2);  // after the two gate/up K slices
        }
      };
      const int n_threads = std::max(1, std::min<int>(16, static_cast<int>(std::thread::hardware_concurrency())));
      std::vector<std::thread> pool;
      for (int t = 0; t < n_threads; ++t)
        pool.emplace_back([&, t]() {
          for (int l = t; l < L; l += n_threads) pack_layer(l);
        });
      for (auto& th : pool) th.join();
      FSX_CUDA_H(cudaMemcpy(h->p_arena, host.data(), total, cudaMemcpyHostToDevice));
      FSX_CUDA_H(cudaMalloc(&h->p_x, static_cast<size_t>(3) * fsx::kTokTile * d * sizeof(float)));
      FSX_CUDA_H(cudaMemset(h->p_x, 0, static_cast<size_t>(3) * fsx::kTokTile * d * sizeof(float)));
      FSX_CUDA_H(cudaMalloc(&h->p_counters, sizeof(int) * (2 * L + 1)));
      h->persist_ok = true;
    }
  }

  // ---- fp32 parameters
  {
    const size_t n_act = static_cast<size_t>(cfg->n_action) * d, n_pos = static_cast<size_t>(T) * d;
    const size_t n_norm = static_cast<size_t>(L) * d;
    std::vector<size_t> sizes = {n_act, n_pos, n_norm, n_norm, static_cast<size_t>(d), static_cast<size_t>(2) * d, 2};
    std::vector<const float*> srcs = {w->act_emb, w->pos_emb, w->attn_norm, w->mlp_norm, w->final_norm, w->head_w, w->head_b};
    size_t total = 0;
    std::vector<size_t> offs;
    for (size_t sz : sizes) {
      offs.push_back(total);
      total += align_up(sz, 64);
    }
    FSX_CUDA_H(cudaMalloc(&h->params, total * sizeof(float)));
    for (size_t i = 0; i < sizes.size(); ++i)
      FSX_CUDA_H(cudaMemcpy(h->params + offs[i], srcs[i], sizes[i] * sizeof(float), cudaMemcpyHostToDevice));
    h->act_emb = h->params + offs[0];
    h->pos_emb = h->params + offs[1];
    h->attn_norm = h->params + offs[2];
    h->mlp_norm = h->params + offs[3];
    h->final_norm = h->params + offs[4];
    h->head_w = h->params + offs[5];
    h->head_b = h->params + offs[6];
  }

  // ---- workspace for max_batch
  const size_t Mmax = static_cast<size_t>(cfg->max_batch) * T;
  const size_t m_pad = (Mmax + 255) / 256 * 256;  // whole token tiles of every GEMM tile size
  FSX_CUDA_H(cudaMalloc(&h->x, m_pad * d * sizeof(float)));
  FSX_CUDA_H(cudaMalloc(&h->x16, m_pad * d * sizeof(__half)));
  h->ss_stride = static_cast<int>(m_pad);
  FSX_CUDA_H(cudaMalloc(&h->ss, static_cast<size_t>(d / 128) * m_pad * sizeof(float)));
  FSX_CUDA_H(cudaMemset(h->ss, 0, static_cast<size_t>(d / 128) * m_pad * sizeof(float)));
  FSX_CUDA_H(cudaMalloc(&h->qkv, m_pad * 3 * HD * sizeof(__half)));
  FSX_CUDA_H(cudaMalloc(&h->o, m_pad * HD * sizeof(__half)));
  FSX_CUDA_H(cudaMalloc(&h->hbuf, m_pad * F * sizeof(__half)));
  FSX_CUDA_H(cudaMemset(h->x16, 0, m_pad * d * sizeof(__half)));
  FSX_CUDA_H(cudaMemset(h->o, 0, m_pad * HD * sizeof(__half)));
  FSX_CUDA_H(cudaMemset(h->hbuf, 0, m_pad * F * sizeof(__half)));
  {
    const uint32_t boxes[4] = {48, 128, 256, 144};
    for (int i = 0; i < 4; ++i) {
      if (!fsx::encode_act_map(&h->map_x16[i], h->x16, m_pad, d, boxes[i]) ||
          !fsx::encode_act_map(&h->map_o[i], h->o, m_pad, HD, boxes[i]) ||
          !fsx::encode_act_map(&h->map_h[i], h->hbuf, m_pad, F, boxes[i]))
        return bail(fail(FSX_ERR_CUDA, "tensor map encoding of the activation buffers failed"));
    }
  }
  size_t part = 0;
  for (int B = 1; B <= cfg->max_batch; ++B)
    part = std::max(part, fsx::attention_workspace_bytes(B, cfg->n_heads, attention_splits(h, B)));
  h->part_bytes = part;
  if (part) FSX_CUDA_H(cudaMalloc(&h->part, part));
  FSX_CUDA_H(cudaMalloc(&h->gemm_part, fsx::gemm_tc_part_bytes(h->sm_count)));
  FSX_CUDA_H(cudaMalloc(&h->tile_count, sizeof(int) * h->sm_count));
  FSX_CUDA_H(cudaMemset(h->tile_count, 0, sizeof(int) * h->sm_count));
  FSX_CUDA_H(cudaMalloc(&h->order, sizeof(int) * cfg->max_batch));
  FSX_CUDA_H(cudaMalloc(&h->plan, sizeof(fsx::AttnPlan) * cfg->max_batch));
  FSX_CUDA_H(cudaMalloc(&h->status, sizeof(int)));
  FSX_CUDA_H(cudaMemset(h->status, 0, sizeof(int)));
  FSX_CUDA_H(cudaMalloc(&h->d_args, sizeof(TickArgs)));
  if (cfg->cache_dtype == FSX_BF16 && cfg->max_total_cache_tokens > 0 && cfg->max_total_cache_tokens <= INT32_MAX) {
    h->h_cache_maps.resize(2 * static_cast<size_t>(cfg->n_layers));
    FSX_CUDA_H(cudaMalloc(&h->d_cache_maps, h->h_cache_maps.size() * sizeof(CUtensorMap)));
  }
  FSX_CUDA_H(cudaMalloc(&h->st_offsets, (cfg->max_batch + 1) * sizeof(int64_t)));
  FSX_CUDA_H(cudaMalloc(&h->st_frames, static_cast<size_t>(cfg->max_batch) * cfg->n_frame * d * sizeof(float) + 16));
  FSX_CUDA_H(cudaMalloc(&h->st_waypoints, static_cast<size_t>(cfg->max_batch) * cfg->n_waypoints * 2 * sizeof(float)));
  FSX_CUDA_H(cudaStreamCreateWithFlags(&h->cap_stream, cudaStreamNonBlocking));
  FSX_CUDA_H(cudaEventCreateWithFlags(&h->last_tick, cudaEventDisableTiming));
  h->tev.resize(2 * static_cast<size_t>(L));
  for (auto& e : h->tev) FSX_CUDA_H(cudaEventCreate(&e));
  FSX_CUDA_H(cudaDeviceSynchronize());
#undef FSX_CUDA_H
  *out = h;
  return FSX_OK;
}

fsx_status fsx_tick_ranges(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                           const int64_t* d_starts, const int64_t* d_offsets, int B, const void* d_frames,
                           float* d_waypoints, void* stream) {
  fsx_status s = check_tick_args(h, k_cache, v_cache, d_offsets, B, d_frames, d_waypoints);
  if (s != FSX_OK) return s;
  std::lock_guard<std::mutex> lock(h->mu);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  s = prepare_tick(h, k_cache, v_cache, d_offsets, d_starts, d_frames, d_waypoints, st);
  if (s != FSX_OK) return s;
  cudaGraphExec_t exec = nullptr;
  s = get_graph(h, B, h->timing, &exec);
  if (s != FSX_OK) return s;
  FSX_CUDA(cudaGraphLaunch(exec, st));
  h->timed_pending = h->timing;
  return finish_tick(h, st);
}

fsx_status fsx_tick(fsx_handle h, const void* const* k_cache, const void* const* v_cache, const int64_t* d_offsets,
                    int B, const void* d_frames, float* d_waypoints, void* stream) {
  return fsx_tick_ranges(h, k_cache, v_cache, nullptr, d_offsets, B, d_frames, d_waypoints, stream);
}

fsx_status fsx_tick_host(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                         const int64_t* h_offsets, int B, const void* h_frames, float* h_waypoints, void* stream) {
  fsx_status s = check_tick_args(h, k_cache, v_cache, h_offsets, B, h_frames, h_waypoints);
  if (s != FSX_OK) return s;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  {
    std::lock_guard<std::mutex> lock(h->mu);
    FSX_CUDA(cudaSetDevice(h->device));
    if (h->has_last && h->last_stream != st) FSX_CUDA(cudaStreamWaitEvent(st, h->last_tick, 0));
    const size_t fbytes = static_cast<size_t>(B) * h->cfg.n_frame * h->cfg.d_model *
                          (h->cfg.frame_dtype == FSX_BF16 ? 2 : 4);
    FSX_CUDA(cudaMemcpyAsync(h->st_offsets, h_offsets, (B + 1) * sizeof(int64_t), cudaMemcpyHostToDevice, st));
    if (fbytes) FSX_CUDA(cudaMemcpyAsync(h->st_frames, h_frames, fbytes, cudaMemcpyHostToDevice, st));
  }
  s = fsx_tick(h, k_cache, v_cache, h->st_offsets, B, h->st_frames, h->st_waypoints, stream);
  if (s != FSX_OK) return s;
  FSX_CUDA(cudaMemcpyAsync(h_waypoints, h->st_waypoints,
                           static_cast<size_t>(B) * h->cfg.n_waypoints * 2 * sizeof(float), cudaMemcpyDeviceToHost, st));
  FSX_CUDA(cudaStreamSynchronize(st));
  return FSX_OK;
}

fsx_status fsx_tick_ranges_debug(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                                 const int64_t* d_starts, const int64_t* d_offsets, int B, const void* d_frames,
                                 float* d_waypoints, void* d_attn_out, void* stream) {
  fsx_status s = check_tick_args(h, k_cache, v_cache, d_offsets, B, d_frames, d_waypoints);
  if (s != FSX_OK) return s;
  if (!d_attn_out) return fail(FSX_ERR_INVALID_ARG, "d_attn_out is NULL");
  std::lock_guard<std::mutex> lock(h->mu);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  s = prepare_tick(h, k_cache, v_cache, d_offsets, d_starts, d_frames, d_waypoints, st);
  if (s != FSX_OK) return s;
  s = enqueue_tick(h, B, st, static_cast<__half*>(d_attn_out), false);
  if (s != FSX_OK) return s;
  return finish_tick(h, st);
}

fsx_status fsx_tick_debug(fsx_handle h, const void* const* k_cache, const void* const* v_cache,
                          const int64_t* d_offsets, int B, const void* d_frames, float* d_waypoints,
                          void* d_attn_out, void* stream) {
  return fsx_tick_ranges_debug(h, k_cache, v_cache, nullptr, d_offsets, B, d_frames, d_waypoints, d_attn_out,
                               stream);
}

// The host reading of the device status word.
static fsx_status status_word(int v) {
  if (v == 0) return FSX_OK;
  if (v == FSX_ERR_TIMEOUT) return fail(FSX_ERR_TIMEOUT, "a device-side wait timed out");
  if (v == FSX_ERR_RANGE) return fail(FSX_ERR_RANGE, "a cache value lies outside the fp16 range");
  return fail(FSX_ERR_DEVICE_ARG, "device-side argument check failed (cache offsets)");
}

fsx_status fsx_get_status(fsx_handle h, void* stream) {
  if (!h) return fail(FSX_ERR_INVALID_ARG, "handle is NULL");
  std::lock_guard<std::mutex> lock(h->mu);
  FSX_CUDA(cudaSetDevice(h->device));
  FSX_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  int v = 0;
  FSX_CUDA(cudaMemcpyAsync(&v, h->status, sizeof(int), cudaMemcpyDeviceToHost, h->cap_stream));
  FSX_CUDA(cudaMemsetAsync(h->status, 0, sizeof(int), h->cap_stream));
  FSX_CUDA(cudaStreamSynchronize(h->cap_stream));
  return status_word(v);
}

void fsx_destroy(fsx_handle h) { free_handle(h); }

fsx_status fsx_set_wait_limit(fsx_handle h, unsigned long long limit_ns) {
  if (!h) return fail(FSX_ERR_INVALID_ARG, "handle is NULL");
  std::lock_guard<std::mutex> lock(h->mu);
  h->wait_limit_ns = limit_ns == 0 ? 1000000000ull : limit_ns;
  // the graphs hold the limit as a kernel argument: capture them again
  for (auto& kv : h->graphs) cudaGraphExecDestroy(kv.second);
  for (auto& kv : h->timed_graphs) cudaGraphExecDestroy(kv.second);
  h->graphs.clear();
  h->timed_graphs.clear();
  return FSX_OK;
}

long long fsx_weight_bytes(fsx_handle h) { return h ? h->weight_bytes : 0; }

int fsx_tick_launches(fsx_handle h, int B) {
  if (!h || B < 1) return 0;
  if (use_persistent(h, B)) return h->paper_head != nullptr ? 2 : 1;
  return 2 + h->cfg.n_layers * (4 + fsx::attention_launch_count(attention_splits(h, B)));
}

fsx_status fsx_set_kernel_timing(fsx_handle h, int enable, int kclass) {
  if (!h) return fail(FSX_ERR_INVALID_ARG, "handle is NULL");
  if (kclass < kClassQkv || kclass > kClassPersistent) return fail(FSX_ERR_INVALID_ARG, "kernel class %d unknown", kclass);
  std::lock_guard<std::mutex> lock(h->mu);
  if (enable && kclass != h->timing_class) {
    for (auto& kv : h->timed_graphs) cudaGraphExecDestroy(kv.second);
    h->timed_graphs.clear();
  }
  h->timing = enable != 0;
  h->timing_class = kclass;
  return FSX_OK;
}

fsx_status fsx_kernel_time(fsx_handle h, float* ms, int* launches) {
  if (!h || !ms || !launches) return fail(FSX_ERR_INVALID_ARG, "NULL argument");
  std::lock_guard<std::mutex> lock(h->mu);
  if (!h->timed_pending || h->timed_pairs == 0) return fail(FSX_ERR_INVALID_ARG, "no timed tick recorded");
  FSX_CUDA(cudaSetDevice(h->device));
  FSX_CUDA(cudaEventSynchronize(h->tev[2 * h->timed_pairs - 1]));
  float total = 0.f;
  for (int i = 0; i < h->timed_pairs; ++i) {
    float t = 0.f;
    FSX_CUDA(cudaEventElapsedTime(&t, h->tev[2 * i], h->tev[2 * i + 1]));
    total += t;
  }
  *ms = total;
  *launches = h->timed_pairs;
  return FSX_OK;
}

size_t fsx_attention_workspace_bytes(int B, int n_heads, int n_q, int n_splits) {
  (void)n_q;
  if (B < 1 || n_heads < 1 || n_splits < 1) return 0;
  return 256 + fsx::attention_workspace_bytes(B, n_heads, n_splits);
}

fsx_status fsx_attention(const void* d_q, long long q_stride, const void* d_k_own, const void* d_v_own,
                         long long own_stride, int n_q, int n_own, const void* d_k_cache, const void* d_v_cache,
                         int cache_dtype, const int64_t* d_offsets, int B, int n_heads, int head_dim, int n_splits,
                         void* d_out, float* d_lse, void* d_workspace, size_t workspace_bytes, void* stream) {
  g_err[0] = '\0';
  if (!d_q || !d_offsets || !d_out) return fail(FSX_ERR_INVALID_ARG, "NULL pointer argument");
  if (n_own > 0 && (!d_k_own || !d_v_own)) return fail(FSX_ERR_INVALID_ARG, "own key/value pointers are NULL");
  if (head_dim != fsx::kHeadDim) return fail(FSX_ERR_UNSUPPORTED, "head_dim must be 128");
  if (n_q < 1 || n_q > fsx::kTokTile) return fail(FSX_ERR_INVALID_ARG, "n_q must be in 1..48");
  if (n_own < 0 || B < 1 || n_heads < 1) return fail(FSX_ERR_INVALID_ARG, "n_own >= 0, B >= 1, n_heads >= 1");
  if (n_splits < 1 || n_splits > fsx::kMaxSplits) return fail(FSX_ERR_INVALID_ARG, "n_splits must be in 1..64");
  if (cache_dtype != FSX_F32 && cache_dtype != FSX_BF16) return fail(FSX_ERR_INVALID_ARG, "bad cache_dtype");
  if (q_stride < static_cast<long long>(n_heads) * head_dim || (n_own > 0 && own_stride < static_cast<long long>(n_heads) * head_dim) ||
      (q_stride % 8) != 0 || (own_stride % 8) != 0)
    return fail(FSX_ERR_INVALID_ARG, "strides must cover n_heads*head_dim and be multiples of 8");
  const size_t need = fsx_attention_workspace_bytes(B, n_heads, n_q, n_splits);
  if (!d_workspace || workspace_bytes < need)
    return fail(FSX_ERR_INVALID_ARG, "workspace of %zu bytes required", need);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int* status = static_cast<int*>(d_workspace);  // first 256 bytes: status word
  float* part = reinterpret_cast<float*>(static_cast<unsigned char*>(d_workspace) + 256);
  FSX_CUDA(cudaMemsetAsync(status, 0, sizeof(int), st));
  FSX_CUDA(fsx::attention_set_attributes());
  fsx::AttnArgs a{};
  a.q = static_cast<const __half*>(d_q);
  a.q_stride = q_stride;
  a.k_own = static_cast<const __half*>(d_k_own);
  a.v_own = static_cast<const __half*>(d_v_own);
  a.own_stride = own_stride;
  a.n_q = n_q;
  a.n_own = n_own;
  a.k_cache = d_k_cache;
  a.v_cache = d_v_cache;
  a.targs = nullptr;
  a.layer = 0;
  a.offsets = d_offsets;
  a.max_total = (1ll << 62);
  a.n_heads = n_heads;
  a.n_splits = n_splits;
  a.out = static_cast<__half*>(d_out);
  a.out_stride = static_cast<long long>(n_heads) * head_dim;
  a.lse = d_lse;
  a.part_o = part;
  a.part_lse = part + static_cast<size_t>(B) * n_heads * n_splits * fsx::kTokTile * fsx::kHeadDim;
  a.status = status;
  FSX_CUDA(fsx::launch_attention(a, B, cache_dtype, st, false));
  return FSX_OK;
}

}  // extern "C"
