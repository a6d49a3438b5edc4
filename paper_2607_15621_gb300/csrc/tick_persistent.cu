// Persistent single-vehicle tick: the whole expert forward (Sec. 3.1, Eq. 1)
// for one vehicle in ONE kernel launch, built for the latency of a B = 1 tick.
//
// Layout of the work: the grid is one thread-block cluster of 4 CTAs per
// attention head (H clusters, 4H CTAs, one CTA per SM, all co-resident).
// Every layer runs two phases separated by device-wide counters:
//   phase A (every cluster = one head h):
//     x -> RMSNorm (each CTA normalises a quarter of the rows and pushes them to
//     its partners through distributed shared memory) -> the CTA's 96 rows of
//     [W_q; W_k; W_v] for head h (32 q, 32 k, 32 v dims) -> q, k_ae, v_ae pushed
//     to all 4 CTAs -> Eq. 1 over a quarter of [K_vlm ; K_ae] per CTA ->
//     the 4 split results merged in shared memory (log-sum-exp weights) ->
//     the CTA's 128 output columns of o_h W_o^T added into the next residual
//     state with vector atomics (cluster 0 also adds the residual itself).
//   phase B (clusters 0 .. F/64-1; cluster c owns SwiGLU columns 64c..64c+63):
//     x -> RMSNorm (split and pushed as above) -> the CTA's 16 SwiGLU columns
//     (gate and up rows side by side) -> h pushed to all 4 CTAs -> the CTA's
//     128 output columns of h W_d^T added into the next residual state.
// The residual stream rotates through three fp32 buffers: a phase reads one,
// accumulates into the next (zeroed one phase earlier) and zeroes the third.
//
// Weights never wait for activations: each CTA's weights are packed in the
// order it consumes them (16 KB chunks, fragment-ordered fp16) and streamed by
// bulk copies through a 6-slot shared-memory ring that is refilled as soon as
// a chunk is consumed, so the HBM stream runs ahead across phases and layers.
// The layer's backbone cache rows are prefetched into L2 at the start of the
// layer and converted bf16/fp32 -> fp16 while staging 32-key tiles.
#include <cooperative_groups.h>
#include <math_constants.h>

#include "device_util.cuh"
#include "kernels.h"
#include "persistent.h"

namespace cg = cooperative_groups;

namespace fsx {

namespace {

constexpr int kThr = kPersistThreads;  // 256 = 8 warps
constexpr int kCl = kPersistCluster;   // 4 CTAs per cluster
constexpr int kSlotBytes = kPersistChunk;
constexpr int kSlots = kPersistSlots;
constexpr int kD = kHeadDim;           // 128
constexpr int kKeyTile = 32;           // keys per staged attention tile
constexpr int kQS = kD + 8;            // fp16 row stride of q / own k / own v / o (halves)
constexpr int kHS = 64 + 8;            // fp16 row stride of the SwiGLU slice (halves)
constexpr int kDS = 128 + 4;           // fp32 row stride of the output transpose buffer
constexpr int kRowsPerRank = kTokTile / kCl;  // 12
constexpr unsigned long long kSpinLimitNs = 1000000000ull;

struct Smem {
  // byte offsets inside the dynamic shared memory
  int full_bar, rstd, ring, act, qbuf, ownk, ownv, tile, recv, recv_lse, total;
};

__host__ __device__ inline Smem smem_layout(int d) {
  Smem s{};
  int o = 0;
  s.full_bar = o;  o += 64;
  s.rstd = o;      o += 256;
  o = 1024;
  s.ring = o;      o += kSlots * kSlotBytes;
  s.act = o;       o += kTokTile * (d + 8) * 2;
  s.qbuf = o;      o += kTokTile * kQS * 2;            // q of this head; later the merged o_h
  s.ownk = o;      o += kTokTile * kQS * 2;            // own keys; later the output transpose
  s.ownv = o;      o += kTokTile * kQS * 2;            // own values
  s.tile = o;      o += 2 * kKeyTile * kD * 2;         // fp16 K|V tile, swizzled
  s.recv = o;      o += kCl * kRowsPerRank * kD * 2;   // fp16 split partials of the rows this CTA merges
  s.recv_lse = o;  o += kCl * kRowsPerRank * 4;
  s.total = o;
  return s;
}

__device__ __forceinline__ int swz(int row, int unit) { return row * 16 + (unit ^ (row & 7)); }

__device__ __forceinline__ float4 ld_cg4(const float* p) { return __ldcg(reinterpret_cast<const float4*>(p)); }

__device__ __forceinline__ void red_add_v4(float* addr, float4 v) {
  asm volatile("red.relaxed.gpu.global.add.v4.f32 [%0], {%1,%2,%3,%4};" ::"l"(addr), "f"(v.x), "f"(v.y), "f"(v.z),
               "f"(v.w)
               : "memory");
}

__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// Device-wide arrival counter: after the CTA barrier one thread adds 1 with
// release semantics, which publishes the CTA's earlier global writes.
__device__ __forceinline__ void arrive(int* counter) {
  __syncthreads();
  if (threadIdx.x == 0) asm volatile("red.release.gpu.global.add.s32 [%0], 1;" ::"l"(counter) : "memory");
}

// Address of the same shared-memory offset in cluster CTA `rank`.
__device__ __forceinline__ uint32_t cluster_addr(const void* local, int rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr(local)), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_cluster_v4(uint32_t addr, uint4 v) {
  asm volatile("st.shared::cluster.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}
__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}

// Copy rows x bytes_per_row (multiple of 16) starting at the same local offset to
// the 3 partner CTAs of the cluster (16-byte remote stores).
__device__ __forceinline__ void push_rows(const void* base, int rows, int row_stride_bytes, int bytes_per_row,
                                          int my_rank, int tid, int nthr) {
  const int upr = bytes_per_row / 16;
  const unsigned char* b = static_cast<const unsigned char*>(base);
  for (int i = tid; i < rows * upr * (kPersistCluster - 1); i += nthr) {
    const int peer_i = i / (rows * upr);
    const int rest = i - peer_i * rows * upr;
    const int r = rest / upr;
    const int u = rest - r * upr;
    const int peer = peer_i + (peer_i >= my_rank ? 1 : 0);
    const unsigned char* src = b + static_cast<size_t>(r) * row_stride_bytes + u * 16;
    st_cluster_v4(cluster_addr(src, peer), *reinterpret_cast<const uint4*>(src));
  }
}

// Bounded wait until *counter >= target (one thread polls, the CTA follows).
// Once any wait of the tick has timed out, later waits return immediately, so
// a broken tick still ends within about a second.
__device__ __forceinline__ void wait_counter(const int* counter, int target, int* status) {
  if (threadIdx.x == 0 && *reinterpret_cast<volatile int*>(status) != kStatusTimeout) {
    const unsigned long long t0 = global_timer_ns();
    for (uint32_t it = 0;; ++it) {
      int v;
      asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(counter) : "memory");
      if (v >= target) break;
      if ((it & 63u) == 63u && global_timer_ns() - t0 > kSpinLimitNs) {
        set_status(status, kStatusTimeout);
        break;
      }
    }
  }
  __syncthreads();
}

// One 16-row weight block (fragment-ordered, kbs k-steps of 16) against the
// 48-token activation tile `act` (row stride `as` halves): acc[token tile][4].
__device__ __forceinline__ void block_gemm(const uint4* w, int kbs, const __half* act, int as, float (&acc)[6][4],
                                           int lane) {
#pragma unroll
  for (int t = 0; t < 6; ++t)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[t][e] = 0.f;
  for (int kb = 0; kb < kbs; kb += 2) {
    uint32_t b[6][2][2];
#pragma unroll
    for (int t = 0; t < 6; ++t) {
      const __half* src = act + static_cast<size_t>(t * 8 + (lane & 7)) * as + kb * 16 + (lane >> 3) * 8;
      ldsm_x4(b[t][0][0], b[t][0][1], b[t][1][0], b[t][1][1], smem_addr(src));
    }
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      const uint4 a = w[(kb + kk) * 32 + lane];
#pragma unroll
      for (int t = 0; t < 6; ++t) mma_f16_16816(acc[t], a.x, a.y, a.z, a.w, b[t][kk][0], b[t][kk][1]);
    }
  }
}

template <typename CT>
__global__ void __cluster_dims__(kCl, 1, 1) __launch_bounds__(kThr, 1) persistent_tick_kernel(const PersistArgs p) {
  extern __shared__ __align__(1024) unsigned char smem[];
  const Smem L = smem_layout(p.d);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.full_bar);
  unsigned char* ring = smem + L.ring;
  __half* act = reinterpret_cast<__half*>(smem + L.act);
  __half* qbuf = reinterpret_cast<__half*>(smem + L.qbuf);
  __half* ownk = reinterpret_cast<__half*>(smem + L.ownk);
  __half* ownv = reinterpret_cast<__half*>(smem + L.ownv);
  uint4* tile_k = reinterpret_cast<uint4*>(smem + L.tile);
  uint4* tile_v = tile_k + kKeyTile * 16;
  __half* recv = reinterpret_cast<__half*>(smem + L.recv);
  float* recv_lse = reinterpret_cast<float*>(smem + L.recv_lse);
  float* dstT = reinterpret_cast<float*>(smem + L.ownk);  // [48][kDS] fp32 output transpose (aliases ownk/ownv)

  cg::cluster_group cluster = cg::this_cluster();
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int rank = static_cast<int>(cluster.block_rank());
  const int head = blockIdx.x / kCl;             // phase A: this cluster's head
  const int G = gridDim.x;
  const int cta = blockIdx.x;
  const int d = p.d;
  const int as = d + 8;
  const int T = p.n_action + p.n_frame;
  const int HD = p.H * kD;
  const bool in_b = head < p.n_b_clusters;       // phase B participant (whole clusters)
  const int n_b_ctas = p.n_b_clusters * kCl;
  const int per_layer = kPersistAChunks + (in_b ? kPersistBChunks : 0);
  const int total_chunks = p.n_layers * per_layer;

  // ---- ring: chunk q of this CTA's stream goes to slot q % kSlots
  auto chunk_src = [&](int q) -> const unsigned char* {
    const int layer = q / per_layer;
    const int i = q - layer * per_layer;
    const unsigned char* base = p.warena + static_cast<size_t>(layer) * p.layer_bytes;
    if (i < kPersistAChunks) return base + static_cast<size_t>(cta) * p.a_cta_bytes + static_cast<size_t>(i) * kSlotBytes;
    return base + p.b_offset + static_cast<size_t>(cta) * p.b_cta_bytes + static_cast<size_t>(i - kPersistAChunks) * kSlotBytes;
  };
  auto issue = [&](int q) {  // called by thread 0 only
    if (q >= total_chunks) return;
    uint64_t* bar = full + (q % kSlots);
    mbar_arrive_expect_tx(bar, kSlotBytes);
    bulk_g2s(ring + static_cast<size_t>(q % kSlots) * kSlotBytes, chunk_src(q), kSlotBytes, bar);
  };
  auto wait_chunk = [&](int q) -> const uint4* {
    mbar_wait(full + (q % kSlots), static_cast<uint32_t>((q / kSlots) & 1), p.status);
    return reinterpret_cast<const uint4*>(ring + static_cast<size_t>(q % kSlots) * kSlotBytes);
  };

  if (tid == 0) {
    for (int i = 0; i < kSlots; ++i) mbar_init(full + i, 1);
    for (int q = 0; q < kSlots; ++q) issue(q);
  }

  // ---- vehicle 0's cache range, checked once (uniform across the grid)
  const int64_t* offs = p.targs->offsets;
  const long long o_lo = offs[0];
  const long long o_hi = offs[1];
  bool bad = o_lo < 0 || o_hi < o_lo || o_hi > p.max_total;
  if (!bad && o_hi > o_lo)  // a non-empty cache needs every layer's rows
    for (int l = 0; l < p.n_layers; ++l)
      bad = bad || p.targs->k_cache[l] == nullptr || p.targs->v_cache[l] == nullptr;
  __syncthreads();
  if (bad) {
    if (cta == 0 && tid == 0) set_status(p.status, kStatusDeviceArg);
    for (int q = 0; q < kSlots && q < total_chunks; ++q) wait_chunk(q);  // let in-flight copies land
    return;
  }
  const long long Lc = o_hi - o_lo;
  const long long n_keys = Lc + T;
  const long long kbeg = n_keys * rank / kCl;
  const long long kend = n_keys * (rank + 1) / kCl;

  float* X0 = p.X;
  const size_t xs = static_cast<size_t>(kTokTile) * d;  // one residual buffer
  const int n_elem = T * d;

  // ---- token assembly: X[0] = [E_act ; F] + P_pos, X[1] = 0
  {
    const int e0 = static_cast<int>(static_cast<long long>(n_elem) * cta / G);
    const int e1 = static_cast<int>(static_cast<long long>(n_elem) * (cta + 1) / G);
    for (int e = e0 + tid; e < e1; e += kThr) {
      const int t = e / d;
      const int c = e - t * d;
      float v;
      if (t < p.n_action) {
        v = p.act_emb[static_cast<size_t>(t) * d + c];
      } else {
        const size_t idx = static_cast<size_t>(t - p.n_action) * d + c;
        v = p.frame_dtype == 1 ? __bfloat162float(static_cast<const __nv_bfloat16*>(p.targs->frames)[idx])
                               : static_cast<const float*>(p.targs->frames)[idx];
      }
      __stcg(X0 + e, v + p.pos_emb[static_cast<size_t>(t) * d + c]);
      __stcg(X0 + xs + e, 0.f);
    }
  }
  arrive(p.counters + 0);

  // x (state buffer) -> RMSNorm -> fp16 rows in every partner's activation tile:
  // this rank normalises rows 12r..12r+11 into its own tile and copies them out
  auto load_normalized = [&](const float* Xs) {
    const int r0 = rank * kRowsPerRank;
    const int r1 = min(r0 + kRowsPerRank, T);
    for (int r = r0 + warp; r < r1; r += kThr / 32) {
      const float* xr = Xs + static_cast<size_t>(r) * d;
      float4 v[8];
      float ss = 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j) {  // lane holds 8 consecutive values per 256-wide slab
        const int c = lane * 8 + j * 256;
        if (c < d) {
          v[2 * j] = ld_cg4(xr + c);
          v[2 * j + 1] = ld_cg4(xr + c + 4);
          ss += v[2 * j].x * v[2 * j].x + v[2 * j].y * v[2 * j].y + v[2 * j].z * v[2 * j].z + v[2 * j].w * v[2 * j].w;
          ss += v[2 * j + 1].x * v[2 * j + 1].x + v[2 * j + 1].y * v[2 * j + 1].y + v[2 * j + 1].z * v[2 * j + 1].z +
                v[2 * j + 1].w * v[2 * j + 1].w;
        }
      }
      ss = warp_sum(ss);
      const float rstd = rsqrtf(ss / static_cast<float>(d) + 1e-6f);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int c = lane * 8 + j * 256;
        if (c < d) {
          uint4 pk;
          pk.x = pack_half2(v[2 * j].x * rstd, v[2 * j].y * rstd);
          pk.y = pack_half2(v[2 * j].z * rstd, v[2 * j].w * rstd);
          pk.z = pack_half2(v[2 * j + 1].x * rstd, v[2 * j + 1].y * rstd);
          pk.w = pack_half2(v[2 * j + 1].z * rstd, v[2 * j + 1].w * rstd);
          *reinterpret_cast<uint4*>(act + static_cast<size_t>(r) * as + c) = pk;
        }
      }
    }
    for (int i = tid; i < (kTokTile - T) * (d / 8); i += kThr) {  // padding token rows
      const int r = T + i / (d / 8);
      *reinterpret_cast<uint4*>(act + static_cast<size_t>(r) * as + (i % (d / 8)) * 8) = make_uint4(0u, 0u, 0u, 0u);
    }
    __syncthreads();
    if (r1 > r0) push_rows(act + static_cast<size_t>(r0) * as, r1 - r0, as * 2, d * 2, rank, tid, kThr);
    cluster.sync();
  };

  // add the CTA's [48 x 128] transposed output (dstT) into X_next columns col0..col0+127,
  // plus the residual X_cur when this is cluster 0
  auto scatter_add = [&](float* Xn, const float* Xc, int col0, bool add_residual) {
    for (int i = tid; i < T * 32; i += kThr) {
      const int t = i >> 5;
      const int c4 = (i & 31) * 4;
      float4 v = *reinterpret_cast<const float4*>(dstT + t * kDS + c4);
      if (add_residual) {
        const float4 r = ld_cg4(Xc + static_cast<size_t>(t) * d + col0 + c4);
        v.x += r.x;
        v.y += r.y;
        v.z += r.z;
        v.w += r.w;
      }
      red_add_v4(Xn + static_cast<size_t>(t) * d + col0 + c4, v);
    }
  };

  // acc (16-row block x 48 tokens) -> dstT rows = tokens, columns col..col+15
  auto store_transposed = [&](const float (&acc)[6][4], int col) {
#pragma unroll
    for (int t = 0; t < 6; ++t) {
      const int m = t * 8 + 2 * (lane & 3);
      const int n = col + (lane >> 2);
      dstT[m * kDS + n] = acc[t][0];
      dstT[(m + 1) * kDS + n] = acc[t][1];
      dstT[m * kDS + n + 8] = acc[t][2];
      dstT[(m + 1) * kDS + n + 8] = acc[t][3];
    }
  };

  int q_chunk = 0;  // next chunk of this CTA's stream to consume
  const float scale_log2 = 1.4426950408889634f * rsqrtf(static_cast<float>(kD));
  const size_t cache_row = static_cast<size_t>(p.H) * kD;  // elements between consecutive tokens

  for (int layer = 0; layer < p.n_layers; ++layer) {
    const int sA = 2 * layer;
    float* Xc = X0 + static_cast<size_t>(sA % 3) * xs;        // layer input
    float* Xm = X0 + static_cast<size_t>((sA + 1) % 3) * xs;  // after attention
    float* Xz = X0 + static_cast<size_t>((sA + 2) % 3) * xs;  // zeroed now, written by phase B
    const CT* kc = static_cast<const CT*>(p.targs->k_cache[layer]);
    const CT* vc = static_cast<const CT*>(p.targs->v_cache[layer]);

    // L2 prefetch of this CTA's cache rows of this layer
    if (warp == 0) {
      const long long c_end = min(kend, Lc);
      for (long long key = kbeg + lane; key < c_end; key += 32) {
        const size_t row = (static_cast<size_t>(o_lo + key) * p.H + head) * kD;
        prefetch_l2(kc + row, kD * sizeof(CT));
        prefetch_l2(vc + row, kD * sizeof(CT));
      }
    }

    // =========================== phase A ===========================
    wait_counter(p.counters + sA, sA == 0 ? G : n_b_ctas, p.status);
    // zero the buffer phase B accumulates into
    {
      const int e0 = static_cast<int>(static_cast<long long>(n_elem) * cta / G);
      const int e1 = static_cast<int>(static_cast<long long>(n_elem) * (cta + 1) / G);
      for (int e = e0 + tid; e < e1; e += kThr) __stcg(Xz + e, 0.f);
    }
    load_normalized(Xc);

    // --- QKV: 6 blocks (q dims 32r..32r+31, then k, then v), one warp each
    if (warp < 6) {
      const uint4* w = wait_chunk(q_chunk + warp);
      float acc[6][4];
      block_gemm(w, d / 16, act, as, acc, lane);
      const int kind = warp >> 1;                       // 0 q, 1 k, 2 v
      const int dim = rank * 32 + (warp & 1) * 16 + (lane >> 2);
      __half* b = kind == 0 ? qbuf : (kind == 1 ? ownk : ownv);
#pragma unroll
      for (int t = 0; t < 6; ++t) {
        const int m = t * 8 + 2 * (lane & 3);
        b[m * kQS + dim] = __float2half_rn(acc[t][0]);
        b[(m + 1) * kQS + dim] = __float2half_rn(acc[t][1]);
        b[m * kQS + dim + 8] = __float2half_rn(acc[t][2]);
        b[(m + 1) * kQS + dim + 8] = __float2half_rn(acc[t][3]);
      }
    }
    __syncthreads();
    if (tid == 0)
      for (int i = 0; i < 6; ++i) issue(q_chunk + i + kSlots);
    q_chunk += 6;
    // this rank's 32 dims of q, k_ae, v_ae (48 rows x 64 bytes each) to the partners
    push_rows(qbuf + rank * 32, kTokTile, kQS * 2, 64, rank, tid, kThr);
    push_rows(ownk + rank * 32, kTokTile, kQS * 2, 64, rank, tid, kThr);
    push_rows(ownv + rank * 32, kTokTile, kQS * 2, 64, rank, tid, kThr);
    cluster.sync();  // q, own k, own v complete in every CTA

    // --- Eq. 1 over keys [kbeg, kend) of [cache ; own], 32-key tiles
    float o_acc[16][4];
    float m_run[2] = {-CUDART_INF_F, -CUDART_INF_F};
    float l_run[2] = {0.f, 0.f};
#pragma unroll
    for (int n = 0; n < 16; ++n)
#pragma unroll
      for (int e = 0; e < 4; ++e) o_acc[n][e] = 0.f;
    uint32_t qf[8][4];
    if (warp < 3) {
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const __half* src = qbuf + static_cast<size_t>(warp * 16 + (lane & 15)) * kQS + kk * 16 + (lane >> 4) * 8;
        ldsm_x4(qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], smem_addr(src));
      }
    }
    const int n_tiles = kend > kbeg ? static_cast<int>((kend - kbeg + kKeyTile - 1) / kKeyTile) : 0;
    // each thread stages 4 of the 1024 16-byte units (K|V x 32 rows x 16 units) of a tile
    uint4 stage[4];
    auto load_tile = [&](int ti) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int u = tid + j * kThr;            // 0..1023
        const int kv = u >> 9;                   // 0 = K, 1 = V
        const int r = (u >> 4) & 31;
        const int c = u & 15;
        const long long key = kbeg + static_cast<long long>(ti) * kKeyTile + r;
        uint4 val = make_uint4(0u, 0u, 0u, 0u);
        if (key < kend) {
          if (key < Lc) {
            const CT* src = (kv ? vc : kc) + (static_cast<size_t>(o_lo + key) * p.H + head) * kD + c * 8;
            if (sizeof(CT) == 2) {
              const uint4 raw = __ldg(reinterpret_cast<const uint4*>(src));
              val = make_uint4(bf16x2_to_half2(raw.x), bf16x2_to_half2(raw.y), bf16x2_to_half2(raw.z),
                               bf16x2_to_half2(raw.w));
            } else {
              const float4 a = __ldg(reinterpret_cast<const float4*>(src));
              const float4 b = __ldg(reinterpret_cast<const float4*>(src) + 1);
              val = make_uint4(pack_half2(a.x, a.y), pack_half2(a.z, a.w), pack_half2(b.x, b.y), pack_half2(b.z, b.w));
            }
          } else {
            const __half* own = (kv ? ownv : ownk) + static_cast<size_t>(key - Lc) * kQS + c * 8;
            val = *reinterpret_cast<const uint4*>(own);
          }
        }
        stage[j] = val;
      }
    };
    auto store_tile = [&]() {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int u = tid + j * kThr;
        const int kv = u >> 9;
        const int r = (u >> 4) & 31;
        const int c = u & 15;
        (kv ? tile_v : tile_k)[swz(r, c)] = stage[j];
      }
    };
    (void)cache_row;
    if (n_tiles > 0) {
      load_tile(0);
      store_tile();
    }
    __syncthreads();
    for (int ti = 0; ti < n_tiles; ++ti) {
      if (ti + 1 < n_tiles) load_tile(ti + 1);  // in flight while the tile is consumed
      if (warp < 3) {
        const int rows = static_cast<int>(min(static_cast<long long>(kKeyTile), kend - kbeg - static_cast<long long>(ti) * kKeyTile));
        float sc[4][4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
#pragma unroll
          for (int e = 0; e < 4; ++e) sc[j][e] = 0.f;
#pragma unroll
          for (int dd = 0; dd < 4; ++dd) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4(b0, b1, b2, b3, smem_addr(tile_k + swz(j * 8 + (lane & 7), dd * 4 + (lane >> 3))));
            mma_f16_16816(sc[j], qf[2 * dd][0], qf[2 * dd][1], qf[2 * dd][2], qf[2 * dd][3], b0, b1);
            mma_f16_16816(sc[j], qf[2 * dd + 1][0], qf[2 * dd + 1][1], qf[2 * dd + 1][2], qf[2 * dd + 1][3], b2, b3);
          }
        }
        float mx[2] = {-CUDART_INF_F, -CUDART_INF_F};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int key = j * 8 + 2 * (lane & 3);
#pragma unroll
          for (int e = 0; e < 4; ++e) sc[j][e] = (key + (e & 1)) < rows ? sc[j][e] * scale_log2 : -CUDART_INF_F;
          mx[0] = fmaxf(mx[0], fmaxf(sc[j][0], sc[j][1]));
          mx[1] = fmaxf(mx[1], fmaxf(sc[j][2], sc[j][3]));
        }
        float alpha[2], m_new[2], rs[2] = {0.f, 0.f};
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
          mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
          m_new[r] = fmaxf(m_run[r], mx[r]);
          alpha[r] = exp2f(m_run[r] - m_new[r]);
          m_run[r] = m_new[r];
        }
        uint32_t pf[2][4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float p0 = exp2f(sc[j][0] - m_new[0]);
          const float p1 = exp2f(sc[j][1] - m_new[0]);
          const float p2 = exp2f(sc[j][2] - m_new[1]);
          const float p3 = exp2f(sc[j][3] - m_new[1]);
          rs[0] += p0 + p1;
          rs[1] += p2 + p3;
          pf[j >> 1][(j & 1) * 2 + 0] = pack_half2(p0, p1);
          pf[j >> 1][(j & 1) * 2 + 1] = pack_half2(p2, p3);
        }
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          rs[r] += __shfl_xor_sync(0xffffffffu, rs[r], 1);
          rs[r] += __shfl_xor_sync(0xffffffffu, rs[r], 2);
          l_run[r] = l_run[r] * alpha[r] + rs[r];
        }
#pragma unroll
        for (int n = 0; n < 16; ++n) {
          o_acc[n][0] *= alpha[0];
          o_acc[n][1] *= alpha[0];
          o_acc[n][2] *= alpha[1];
          o_acc[n][3] *= alpha[1];
        }
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
#pragma unroll
          for (int np = 0; np < 8; ++np) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4_trans(b0, b1, b2, b3,
                          smem_addr(tile_v + swz(kk * 16 + (lane & 7) + 8 * ((lane >> 3) & 1), np * 2 + (lane >> 4))));
            mma_f16_16816(o_acc[2 * np], pf[kk][0], pf[kk][1], pf[kk][2], pf[kk][3], b0, b1);
            mma_f16_16816(o_acc[2 * np + 1], pf[kk][0], pf[kk][1], pf[kk][2], pf[kk][3], b2, b3);
          }
        }
      }
      __syncthreads();  // tile consumed
      if (ti + 1 < n_tiles) {
        store_tile();
        __syncthreads();
      }
    }

    // --- merge the 4 splits: stage this split's normalised partial (fp16) and
    // log-sum-exp locally, then send each row to the rank that owns it
    __half* part = reinterpret_cast<__half*>(tile_k);  // [48][kD] (tile area, free now)
    float* part_lse = reinterpret_cast<float*>(smem + L.rstd);
    if (warp < 3) {
      const int qr0 = warp * 16 + (lane >> 2);
      const int qr1 = qr0 + 8;
      const float inv0 = l_run[0] > 0.f ? 1.f / l_run[0] : 0.f;
      const float inv1 = l_run[1] > 0.f ? 1.f / l_run[1] : 0.f;
#pragma unroll
      for (int n = 0; n < 16; ++n) {
        const int c = n * 8 + 2 * (lane & 3);
        *reinterpret_cast<uint32_t*>(part + qr0 * kD + c) = pack_half2(o_acc[n][0] * inv0, o_acc[n][1] * inv0);
        *reinterpret_cast<uint32_t*>(part + qr1 * kD + c) = pack_half2(o_acc[n][2] * inv1, o_acc[n][3] * inv1);
      }
      if ((lane & 3) == 0) {
        part_lse[qr0] = l_run[0] > 0.f ? m_run[0] + log2f(l_run[0]) : -CUDART_INF_F;
        part_lse[qr1] = l_run[1] > 0.f ? m_run[1] + log2f(l_run[1]) : -CUDART_INF_F;
      }
    }
    __syncthreads();
    for (int i = tid; i < kTokTile * (kD / 8); i += kThr) {  // 48 rows x 16 units
      const int row = i / (kD / 8);
      const int u = i - row * (kD / 8);
      const int owner = row / kRowsPerRank;
      const __half* src = part + row * kD + u * 8;
      st_cluster_v4(cluster_addr(recv + (rank * kRowsPerRank + row - owner * kRowsPerRank) * kD + u * 8, owner),
                    *reinterpret_cast<const uint4*>(src));
    }
    if (tid < kTokTile) {
      const int owner = tid / kRowsPerRank;
      st_cluster_f32(cluster_addr(recv_lse + rank * kRowsPerRank + tid - owner * kRowsPerRank, owner), part_lse[tid]);
    }
    cluster.sync();
    // merged rows of o_h -> every partner's qbuf (now free) as the W_o input
    {
      const int r0 = rank * kRowsPerRank;
      for (int i = tid; i < kRowsPerRank * (kD / 4); i += kThr) {
        const int rr = i / (kD / 4);
        const int row = r0 + rr;
        const int c = (i % (kD / 4)) * 4;
        float mmax = -CUDART_INF_F;
#pragma unroll
        for (int s = 0; s < kCl; ++s) mmax = fmaxf(mmax, recv_lse[s * kRowsPerRank + rr]);
        float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f, wsum = 0.f;
        if (mmax != -CUDART_INF_F) {
#pragma unroll
          for (int s = 0; s < kCl; ++s) {
            const float w = exp2f(recv_lse[s * kRowsPerRank + rr] - mmax);
            const uint2 pk = *reinterpret_cast<const uint2*>(recv + (s * kRowsPerRank + rr) * kD + c);
            const float2 f0 = __half22float2(*reinterpret_cast<const __half2*>(&pk.x));
            const float2 f1 = __half22float2(*reinterpret_cast<const __half2*>(&pk.y));
            a0 += w * f0.x;
            a1 += w * f0.y;
            a2 += w * f1.x;
            a3 += w * f1.y;
            wsum += w;
          }
        }
        const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
        uint2 out;
        out.x = pack_half2(a0 * inv, a1 * inv);
        out.y = pack_half2(a2 * inv, a3 * inv);
        *reinterpret_cast<uint2*>(qbuf + row * kQS + c) = out;
        if (p.attn_capture != nullptr && row < T)
          *reinterpret_cast<uint2*>(p.attn_capture + (static_cast<size_t>(layer) * T + row) * HD + head * kD + c) = out;
      }
    }
    __syncthreads();
    push_rows(qbuf + rank * kRowsPerRank * kQS, kRowsPerRank, kQS * 2, kD * 2, rank, tid, kThr);
    cluster.sync();  // o_h complete everywhere; ownk/ownv free for the transpose

    // --- W_o: this CTA's 128 output columns for head h (8 blocks, one per warp)
    {
      const uint4* w = wait_chunk(q_chunk + (warp >> 2)) + (warp & 3) * (kD / 16) * 32;
      float acc[6][4];
      block_gemm(w, kD / 16, qbuf, kQS, acc, lane);
      store_transposed(acc, warp * 16);
    }
    __syncthreads();
    if (tid == 0)
      for (int i = 0; i < 2; ++i) issue(q_chunk + i + kSlots);
    q_chunk += 2;
    scatter_add(Xm, Xc, rank * 128, head == 0);
    arrive(p.counters + sA + 1);

    // =========================== phase B ===========================
    if (in_b) {
      const int c = head;  // SwiGLU column block 64c..64c+63
      wait_counter(p.counters + sA + 1, G, p.status);
      {  // zero the buffer the next phase A accumulates into (this layer's input is consumed)
        const int e0 = static_cast<int>(static_cast<long long>(n_elem) * cta / n_b_ctas);
        const int e1 = static_cast<int>(static_cast<long long>(n_elem) * (cta + 1) / n_b_ctas);
        for (int e = e0 + tid; e < e1; e += kThr) __stcg(Xc + e, 0.f);
      }
      load_normalized(Xm);
      __half* hsl = qbuf;  // [48][kHS] SwiGLU slice of this cluster
      if (warp < 2) {     // 2 blocks: 8 gate + 8 up rows each -> 8 SwiGLU columns each
        const uint4* w = wait_chunk(q_chunk + warp);
        float acc[6][4];
        block_gemm(w, d / 16, act, as, acc, lane);
        const int col = rank * 16 + warp * 8 + (lane >> 2);
#pragma unroll
        for (int t = 0; t < 6; ++t) {
          const int m = t * 8 + 2 * (lane & 3);
          const float h0 = acc[t][0] / (1.f + __expf(-acc[t][0])) * acc[t][2];
          const float h1 = acc[t][1] / (1.f + __expf(-acc[t][1])) * acc[t][3];
          hsl[m * kHS + col] = __float2half_rn(h0);
          hsl[(m + 1) * kHS + col] = __float2half_rn(h1);
        }
      }
      __syncthreads();
      if (tid == 0)
        for (int i = 0; i < 2; ++i) issue(q_chunk + i + kSlots);
      q_chunk += 2;
      push_rows(hsl + rank * 16, kTokTile, kHS * 2, 32, rank, tid, kThr);
      cluster.sync();  // SwiGLU slice complete everywhere
      {
        const uint4* w = wait_chunk(q_chunk) + warp * (64 / 16) * 32;
        float acc[6][4];
        block_gemm(w, 64 / 16, hsl, kHS, acc, lane);
        store_transposed(acc, warp * 16);
      }
      __syncthreads();
      if (tid == 0) issue(q_chunk + kSlots);
      q_chunk += 1;
      float* Xn = X0 + static_cast<size_t>((sA + 2) % 3) * xs;
      scatter_add(Xn, Xm, rank * 128, c == 0);
      arrive(p.counters + sA + 2);
      (void)c;
    }
  }

  // =========================== head ===========================
  if (cta == 0) {
    wait_counter(p.counters + 2 * p.n_layers, n_b_ctas, p.status);
    const float* Xf = X0 + static_cast<size_t>((2 * p.n_layers) % 3) * xs;
    for (int j = warp; j < p.n_waypoints; j += kThr / 32) {
      const float* xr = Xf + static_cast<size_t>(j) * d;
      float ss = 0.f;
      for (int c = lane; c < d; c += 32) {
        const float v = __ldcg(xr + c);
        ss += v * v;
      }
      ss = warp_sum(ss);
      const float rstd = rsqrtf(ss / static_cast<float>(d) + 1e-6f);
      float o0 = 0.f, o1 = 0.f;
      for (int c = lane; c < d; c += 32) {
        const float n = __ldcg(xr + c) * rstd * p.final_norm[c];
        o0 += p.head_w[c] * n;
        o1 += p.head_w[d + c] * n;
      }
      o0 = warp_sum(o0);
      o1 = warp_sum(o1);
      if (lane == 0) {
        p.targs->waypoints[j * 2 + 0] = o0 + p.head_b[0];
        p.targs->waypoints[j * 2 + 1] = o1 + p.head_b[1];
      }
    }
  }
}

}  // namespace

size_t persistent_smem_bytes(int d) { return static_cast<size_t>(smem_layout(d).total); }

cudaError_t persistent_set_attributes(int d) {
  const int bytes = static_cast<int>(persistent_smem_bytes(d));
  cudaError_t e = cudaFuncSetAttribute(reinterpret_cast<const void*>(&persistent_tick_kernel<__nv_bfloat16>),
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(reinterpret_cast<const void*>(&persistent_tick_kernel<float>),
                              cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

int persistent_max_clusters(int d, int cache_dtype) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kCl * 64);
  cfg.blockDim = dim3(kThr);
  cfg.dynamicSmemBytes = persistent_smem_bytes(d);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCl;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  const void* fn = cache_dtype == 1 ? reinterpret_cast<const void*>(&persistent_tick_kernel<__nv_bfloat16>)
                                   : reinterpret_cast<const void*>(&persistent_tick_kernel<float>);
  if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) == cudaSuccess) return n;
  cudaGetLastError();
  cfg.numAttrs = 0;  // the cluster shape is compiled into the kernel
  if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) == cudaSuccess) return n;
  cudaGetLastError();
  return 0;
}

cudaError_t launch_persistent(const PersistArgs& a_in, int cache_dtype, cudaStream_t stream) {
  PersistArgs a = a_in;
  void* kargs[] = {&a};
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kCl * a.H);
  cfg.blockDim = dim3(kThr);
  cfg.dynamicSmemBytes = persistent_smem_bytes(a.d);
  cfg.stream = stream;
  cfg.numAttrs = 0;  // cluster shape comes from __cluster_dims__
  const void* fn = cache_dtype == 1 ? reinterpret_cast<const void*>(&persistent_tick_kernel<__nv_bfloat16>)
                                    : reinterpret_cast<const void*>(&persistent_tick_kernel<float>);
  return cudaLaunchKernelExC(&cfg, fn, kargs);
}

}  // namespace fsx
