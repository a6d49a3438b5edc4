// Eq. 1 of Sec. 3.1: the expert's queries of one vehicle and one head attend,
// with a single softmax, over the concatenation [K_vlm ; K_ae] / [V_vlm ; V_ae]
// of that layer's backbone cache rows (read only) and the expert's own keys and
// values. No mask, no rotary phase on the expert side, scale 1/sqrt(128).
//
// Split-KV flash decoding: the L_b + T keys of a vehicle are cut into
// n_splits near-equal ranges; one CTA (3 warps x 16 queries = 48 query rows)
// streams its range in 32-key chunks. Each chunk is staged raw (bf16 / fp32 cache
// rows, fp16 own rows) with 16-byte cp.async, converted once to fp16 into an
// XOR-swizzled tile, and the next chunk is issued into the raw buffer while the
// tile is consumed by mma.sync m16n8k16 (S = Q K^T with the query fragments read
// from a shared tile, then O += P V with P kept in registers) under an online
// softmax in the log2 domain. With one split the CTA writes the normalised output.
// With 2..8 splits the splits of one (vehicle, head) form a thread-block
// cluster: each CTA leaves (O / l, m + log2 l) in its shared memory and, after
// a cluster barrier, merges a slice of the query rows over all splits through
// distributed shared memory (lse = log2 sum_s 2^lse_s, o = sum_s
// 2^(lse_s - lse) o_s), in split order. More splits fall back to global
// partials merged by a second kernel.
#include <cooperative_groups.h>
#include <math_constants.h>

#include "device_util.cuh"
#include "kernels.h"

namespace cg = cooperative_groups;

namespace fsx {

namespace {

constexpr int kMaxClusterSplits = 8;
constexpr int kWarps = 3;
constexpr int kThreads = kWarps * 32;
#ifndef FSX_ATTN_CHUNK
#define FSX_ATTN_CHUNK 32
#endif
#ifndef FSX_ATTN_MIN_CTAS
#define FSX_ATTN_MIN_CTAS 5
#endif
#ifndef FSX_ATTN_RAW_STAGES
#define FSX_ATTN_RAW_STAGES 1
#endif
constexpr int kChunk = FSX_ATTN_CHUNK;  // keys per staged chunk
constexpr int kRawStages = FSX_ATTN_RAW_STAGES;  // raw chunks staged (in flight while one is computed)
constexpr int kNT = kChunk / 8;         // 8-key n tiles of S
constexpr int kKS = kChunk / 16;        // 16-key k steps of P V
constexpr int kD = kHeadDim;           // 128
constexpr int kUnits = kD * 2 / 16;    // 16-byte units per fp16 row (16)

template <typename CT>
struct CacheRow {
  static constexpr int kBytes = kD * static_cast<int>(sizeof(CT));
};

// raw staging: [kRawStages][K|V][kChunk rows][row bytes]; compute tiles: fp16 [K|V][kChunk][kD] swizzled
// The CTA's 48 query rows stay in shared memory and their fragments are re-read for
// every chunk: that keeps the register budget at 128, so 5 CTAs (15 warps) share an SM.
constexpr size_t kQTileBytes = static_cast<size_t>(kTokTile) * kD * 2;

template <typename CT>
__host__ __device__ constexpr size_t attn_smem_bytes() {
  return static_cast<size_t>(kRawStages) * 2 * kChunk * CacheRow<CT>::kBytes + static_cast<size_t>(2) * kChunk * kD * 2 +
         kQTileBytes;
}

__device__ __forceinline__ int swz(int row, int unit) { return row * kUnits + (unit ^ (row & 7)); }

// 2^x on the special-function unit (relative error about 2^-22; -inf -> +0)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// The running maximum is only moved when a row's chunk maximum exceeds it by more
// than this (log2 units), so P <= 2^8 stays well inside fp16 and the rescale of the
// accumulators is skipped for most chunks; the result does not depend on it.
constexpr float kLazyRescale = 8.f;

// wait until at most n of this thread's cp.async groups are pending
__device__ __forceinline__ void cp_async_wait_n(int n) {
  if (n <= 0) cp_async_wait<0>();
  else if (n == 1) cp_async_wait<1>();
  else if (n == 2) cp_async_wait<2>();
  else cp_async_wait<3>();
}

template <typename CT>
__device__ __forceinline__ void convert_unit(const unsigned char* raw, uint4* dst, bool own, uint32_t& range);

// bf16 cache rows: 16 raw bytes = 8 values -> 8 fp16 (saturated, out-of-range values recorded)
template <>
__device__ __forceinline__ void convert_unit<__nv_bfloat16>(const unsigned char* raw, uint4* dst, bool own,
                                                            uint32_t& range) {
  const uint4 v = *reinterpret_cast<const uint4*>(raw);
  if (own) {
    *dst = v;
  } else {
    *dst = make_uint4(bf16x2_to_half2_sat(v.x, range), bf16x2_to_half2_sat(v.y, range),
                      bf16x2_to_half2_sat(v.z, range), bf16x2_to_half2_sat(v.w, range));
  }
}

// fp32 cache rows: 32 raw bytes = 8 values -> 8 fp16 (own rows are fp16 in the first half)
template <>
__device__ __forceinline__ void convert_unit<float>(const unsigned char* raw, uint4* dst, bool own, uint32_t& range) {
  if (own) {
    *dst = *reinterpret_cast<const uint4*>(raw);
  } else {
    const float4 a = *reinterpret_cast<const float4*>(raw);
    const float4 b = *reinterpret_cast<const float4*>(raw + 16);
    *dst = make_uint4(f32x2_to_half2_sat(a.x, a.y, range), f32x2_to_half2_sat(a.z, a.w, range),
                      f32x2_to_half2_sat(b.x, b.y, range), f32x2_to_half2_sat(b.z, b.w, range));
  }
}

static_assert((kTokTile + kMaxClusterSplits - 1) * (kD + 1) * 4 <= (2 * kRawStages + 2) * kChunk * kD * 2 + kQTileBytes,
              "the cluster merge buffers must fit in the staging memory");

template <typename CT, bool CM>
__global__ void __launch_bounds__(kThreads, FSX_ATTN_MIN_CTAS) attn_splitkv_kernel(const AttnArgs p) {
  extern __shared__ __align__(128) unsigned char smem[];
  constexpr int RB = CacheRow<CT>::kBytes;
  unsigned char* raw = smem;                                              // [kRawStages][2][kChunk][RB]
  uint4* tile = reinterpret_cast<uint4*>(smem + static_cast<size_t>(kRawStages) * 2 * kChunk * RB);
  uint4* kt = tile;                      // fp16 K chunk, swizzled
  uint4* vt = tile + kChunk * kUnits;    // fp16 V chunk, swizzled

  const int split = blockIdx.x;
  const int h = blockIdx.y;
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int H = p.n_heads;

  pdl_launch_dependents();
  pdl_wait();
  const int b = p.order != nullptr ? p.order[blockIdx.z] : static_cast<int>(blockIdx.z);
  // The CTAs of a merge cluster read each other's shared memory, so they must
  // all stay; a raised status is honoured per vehicle below instead.
  if (!CM && *reinterpret_cast<volatile int*>(p.status) != 0) return;

  const CT* kc;
  const CT* vc;
  const int64_t* offs;
  const int64_t* starts = nullptr;
  if (p.targs != nullptr) {
    kc = static_cast<const CT*>(p.targs->k_cache[p.layer]);
    vc = static_cast<const CT*>(p.targs->v_cache[p.layer]);
    offs = p.targs->offsets;
    starts = p.targs->starts;
  } else {
    kc = static_cast<const CT*>(p.k_cache);
    vc = static_cast<const CT*>(p.v_cache);
    offs = p.offsets;
  }
  const long long o_lo = starts != nullptr ? starts[b] : offs[b];
  const long long o_hi = o_lo + (offs[b + 1] - offs[b]);
  if (o_lo < 0 || o_hi < o_lo || o_hi > p.max_total ||
      (o_hi > o_lo && (kc == nullptr || vc == nullptr))) {  // never read outside the caller's cache
    set_status(p.status, kStatusDeviceArg);
    return;
  }
  const long long L = o_hi - o_lo;
  const long long n_keys = L + p.n_own;
  const long long kbeg = n_keys * split / p.n_splits;
  const long long kend = n_keys * (split + 1) / p.n_splits;

  // output slots
  const size_t part_base = (static_cast<size_t>(b) * H + h) * p.n_splits + split;  // partial index

  const bool empty_range = kend <= kbeg;
  if (empty_range && !CM) {  // an empty key range contributes nothing
    if (p.n_splits > 1) {
      for (int i = tid; i < kTokTile; i += kThreads) p.part_lse[part_base * kTokTile + i] = -CUDART_INF_F;
      float* po = p.part_o + part_base * kTokTile * kD;
      for (int i = tid; i < kTokTile * kD; i += kThreads) po[i] = 0.f;
    } else {
      for (int i = tid; i < p.n_q * kD; i += kThreads) {
        const int qi = i / kD;
        const int d = i % kD;
        p.out[(static_cast<size_t>(b) * p.n_q + qi) * p.out_stride + h * kD + d] = __float2half_rn(0.f);
      }
      if (p.lse != nullptr)
        for (int i = tid; i < p.n_q; i += kThreads) p.lse[(static_cast<size_t>(b) * H + h) * p.n_q + i] = -CUDART_INF_F;
    }
    return;
  }

  // ---- stage chunk c (keys kbeg + kChunk c ...) into raw stage s
  constexpr int UPR = RB / 16;               // 16-byte units per raw row
  constexpr int RPP = kThreads / UPR;        // raw rows per pass of the CTA
  constexpr int RAW_PASSES = (kChunk + RPP - 1) / RPP;
  static_assert(kThreads % UPR == 0, "whole raw rows per pass");
  const int su = tid % UPR;
  const int sr = tid / UPR;
  const size_t tok_bytes = static_cast<size_t>(H) * RB;  // bytes between two tokens of one head
  const unsigned char* kbase =
      reinterpret_cast<const unsigned char*>(kc) + (static_cast<size_t>(o_lo) * H + h) * RB + su * 16;
  const unsigned char* vbase =
      reinterpret_cast<const unsigned char*>(vc) + (static_cast<size_t>(o_lo) * H + h) * RB + su * 16;
  auto issue_chunk = [&](int c, int s) {
    const long long c0 = kbeg + static_cast<long long>(c) * kChunk;
    const int rows = static_cast<int>(min(static_cast<long long>(kChunk), kend - c0));
    unsigned char* kr = raw + (static_cast<size_t>(s) * 2 + 0) * kChunk * RB;
    unsigned char* vr = raw + (static_cast<size_t>(s) * 2 + 1) * kChunk * RB;
    if (c0 + kChunk <= L) {  // cache rows only: fixed (row, unit) per thread
      const size_t g = static_cast<size_t>(c0 + sr) * tok_bytes;
      const unsigned char* ks = kbase + g;
      const unsigned char* vs = vbase + g;
      const uint32_t kd = smem_addr(kr + sr * RB + su * 16);
      const uint32_t vd = smem_addr(vr + sr * RB + su * 16);
#pragma unroll
      for (int k = 0; k < RAW_PASSES; ++k) {
        if (sr + k * RPP < rows) {
          cp_async_16(kd + k * RPP * RB, ks + k * RPP * tok_bytes);
          cp_async_16(vd + k * RPP * RB, vs + k * RPP * tok_bytes);
        }
      }
      cp_async_commit();
      return;
    }
    for (int i = tid; i < rows * UPR; i += kThreads) {
      const int r = i / UPR;
      const int u = i - r * UPR;
      const long long key = c0 + r;
      const void* ks;
      const void* vs;
      if (key < L) {
        const size_t row = (static_cast<size_t>(o_lo + key) * H + h) * kD;
        ks = reinterpret_cast<const unsigned char*>(kc + row) + u * 16;
        vs = reinterpret_cast<const unsigned char*>(vc + row) + u * 16;
      } else {
        if (u * 16 >= kD * 2) continue;  // own rows are fp16 (256 bytes)
        const size_t row = (static_cast<size_t>(b) * p.n_own + static_cast<size_t>(key - L)) * p.own_stride + h * kD;
        ks = reinterpret_cast<const unsigned char*>(p.k_own + row) + u * 16;
        vs = reinterpret_cast<const unsigned char*>(p.v_own + row) + u * 16;
      }
      cp_async_16(smem_addr(kr + static_cast<size_t>(r) * RB + u * 16), ks);
      cp_async_16(smem_addr(vr + static_cast<size_t>(r) * RB + u * 16), vs);
    }
    cp_async_commit();
  };

  // ---- Q fragments (A operand, 16 queries x 128) straight from global
  const int qr0 = warp * 16 + (lane >> 2);
  const int qr1 = qr0 + 8;
  uint4* qt = tile + 2 * kChunk * kUnits;  // [kTokTile][kD] fp16 queries, swizzled
  for (int i = tid; i < kTokTile * kUnits; i += kThreads) {
    const int r = i / kUnits;
    const int u = i - r * kUnits;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (r < p.n_q)
      v = *reinterpret_cast<const uint4*>(p.q + (static_cast<size_t>(b) * p.n_q + r) * p.q_stride + h * kD + u * 8);
    qt[swz(r, u)] = v;  // made visible by the first chunk's barrier
  }

  float o_acc[16][4];
#pragma unroll
  for (int n = 0; n < 16; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) o_acc[n][e] = 0.f;
  float m_run[2] = {-CUDART_INF_F, -CUDART_INF_F};
  float l_run[2] = {0.f, 0.f};
  const float scale_log2 = 1.4426950408889634f * rsqrtf(static_cast<float>(kD));

  const int n_chunks = empty_range ? 0 : static_cast<int>((kend - kbeg + kChunk - 1) / kChunk);
  for (int i = 0; i < kRawStages && i < n_chunks; ++i) issue_chunk(i, i);
  uint32_t range = 0;  // a cache value outside the fp16 range was saturated

  for (int c = 0; c < n_chunks; ++c) {
    const int s = c % kRawStages;
    cp_async_wait_n(min(kRawStages - 1, n_chunks - 1 - c));  // chunk c landed
    __syncthreads();  // raw stage s complete for everyone; previous tile consumers done

    // ---- convert raw stage s -> fp16 swizzled tiles (rows beyond the range are zero)
    const long long c0 = kbeg + static_cast<long long>(c) * kChunk;
    const int rows = static_cast<int>(min(static_cast<long long>(kChunk), kend - c0));
    {
      const unsigned char* kr = raw + (static_cast<size_t>(s) * 2 + 0) * kChunk * RB;
      const unsigned char* vr = raw + (static_cast<size_t>(s) * 2 + 1) * kChunk * RB;
      constexpr int SRC_UNIT = RB / kUnits;  // raw bytes per 16-byte fp16 unit
      constexpr int TPP = kThreads / kUnits;  // tile rows per pass
      static_assert(kThreads % kUnits == 0, "whole tile rows per pass");
      if (c0 + kChunk <= L) {  // cache rows only
        const int u = tid % kUnits;
#pragma unroll
        for (int k = 0; k < (kChunk + TPP - 1) / TPP; ++k) {
          const int r = tid / kUnits + k * TPP;
          if (r < kChunk) {
            uint4* kd = kt + swz(r, u);
            uint4* vd = vt + swz(r, u);
            if (r < rows) {
              convert_unit<CT>(kr + static_cast<size_t>(r) * RB + u * SRC_UNIT, kd, false, range);
              convert_unit<CT>(vr + static_cast<size_t>(r) * RB + u * SRC_UNIT, vd, false, range);
            } else {
              *kd = make_uint4(0u, 0u, 0u, 0u);
              *vd = make_uint4(0u, 0u, 0u, 0u);
            }
          }
        }
      } else for (int i = tid; i < kChunk * kUnits; i += kThreads) {
        const int r = i / kUnits;
        const int u = i - r * kUnits;
        uint4* kd = kt + swz(r, u);
        uint4* vd = vt + swz(r, u);
        if (r < rows) {
          const bool own = (c0 + r) >= L;
          const int off = own ? u * 16 : u * SRC_UNIT;
          convert_unit<CT>(kr + static_cast<size_t>(r) * RB + off, kd, own, range);
          convert_unit<CT>(vr + static_cast<size_t>(r) * RB + off, vd, own, range);
        } else {
          *kd = make_uint4(0u, 0u, 0u, 0u);
          *vd = make_uint4(0u, 0u, 0u, 0u);
        }
      }
    }
    __syncthreads();  // tiles ready, raw stage s free
    if (c + kRawStages < n_chunks) issue_chunk(c + kRawStages, s);

    // ---- S = Q K^T for 16 queries x kChunk keys
    float sc[kNT][4];
#pragma unroll
    for (int j = 0; j < kNT; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) sc[j][e] = 0.f;
    }
#pragma unroll
    for (int dd = 0; dd < 4; ++dd) {  // 32 dims per ldmatrix.x4
      uint32_t qa[2][4];  // A fragments of the two 16-dim k steps
      const int qrow = warp * 16 + (lane & 15);
#pragma unroll
      for (int t = 0; t < 2; ++t)
        ldsm_x4(qa[t][0], qa[t][1], qa[t][2], qa[t][3], smem_addr(qt + swz(qrow, (2 * dd + t) * 2 + (lane >> 4))));
#pragma unroll
      for (int j = 0; j < kNT; ++j) {
        const int row = j * 8 + (lane & 7);
        const int unit = dd * 4 + (lane >> 3);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(b0, b1, b2, b3, smem_addr(kt + swz(row, unit)));
        mma_f16_16816(sc[j], qa[0][0], qa[0][1], qa[0][2], qa[0][3], b0, b1);
        mma_f16_16816(sc[j], qa[1][0], qa[1][1], qa[1][2], qa[1][3], b2, b3);
      }
    }
    // ---- online softmax (log2 domain; the 1/sqrt(d) log2(e) scale is applied inside
    // the exponent), masking keys past the range on a ragged chunk only
    if (rows < kChunk) {
#pragma unroll
      for (int j = 0; j < kNT; ++j) {
        const int key = j * 8 + 2 * (lane & 3);
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (key + (e & 1) >= rows) sc[j][e] = -CUDART_INF_F;
      }
    }
    float mx[2] = {-CUDART_INF_F, -CUDART_INF_F};
#pragma unroll
    for (int j = 0; j < kNT; ++j) {
      mx[0] = fmaxf(mx[0], fmaxf(sc[j][0], sc[j][1]));
      mx[1] = fmaxf(mx[1], fmaxf(sc[j][2], sc[j][3]));
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
      mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
      mx[r] *= scale_log2;
    }
    if (__any_sync(0xffffffffu, mx[0] > m_run[0] + kLazyRescale || mx[1] > m_run[1] + kLazyRescale)) {
      float alpha[2];
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const float m_new = fmaxf(m_run[r], mx[r]);
        alpha[r] = ex2_approx(m_run[r] - m_new);
        m_run[r] = m_new;
        l_run[r] *= alpha[r];
      }
#pragma unroll
      for (int n = 0; n < 16; ++n) {
        o_acc[n][0] *= alpha[0];
        o_acc[n][1] *= alpha[0];
        o_acc[n][2] *= alpha[1];
        o_acc[n][3] *= alpha[1];
      }
    }
    const float nm0 = -m_run[0];
    const float nm1 = -m_run[1];
    float rs[2] = {0.f, 0.f};
    uint32_t pf[kKS][4];  // P as A fragments, one per k16 step of 16 keys
#pragma unroll
    for (int j = 0; j < kNT; ++j) {
      const float p0 = ex2_approx(fmaf(sc[j][0], scale_log2, nm0));
      const float p1 = ex2_approx(fmaf(sc[j][1], scale_log2, nm0));
      const float p2 = ex2_approx(fmaf(sc[j][2], scale_log2, nm1));
      const float p3 = ex2_approx(fmaf(sc[j][3], scale_log2, nm1));
      rs[0] += p0 + p1;
      rs[1] += p2 + p3;
      const int kk = j >> 1;
      if ((j & 1) == 0) {
        pf[kk][0] = pack_half2(p0, p1);
        pf[kk][1] = pack_half2(p2, p3);
      } else {
        pf[kk][2] = pack_half2(p0, p1);
        pf[kk][3] = pack_half2(p2, p3);
      }
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      rs[r] += __shfl_xor_sync(0xffffffffu, rs[r], 1);
      rs[r] += __shfl_xor_sync(0xffffffffu, rs[r], 2);
      l_run[r] += rs[r];
    }
    // ---- O += P V
#pragma unroll
    for (int kk = 0; kk < kKS; ++kk) {
#pragma unroll
      for (int np = 0; np < 8; ++np) {  // pairs of 8-wide d tiles
        const int row = kk * 16 + (lane & 7) + 8 * ((lane >> 3) & 1);
        const int unit = np * 2 + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_trans(b0, b1, b2, b3, smem_addr(vt + swz(row, unit)));
        mma_f16_16816(o_acc[2 * np], pf[kk][0], pf[kk][1], pf[kk][2], pf[kk][3], b0, b1);
        mma_f16_16816(o_acc[2 * np + 1], pf[kk][0], pf[kk][1], pf[kk][2], pf[kk][3], b2, b3);
      }
    }
  }
  flag_range(p.status, range);

  // ---- write out
  const float inv0 = l_run[0] > 0.f ? 1.f / l_run[0] : 0.f;
  const float inv1 = l_run[1] > 0.f ? 1.f / l_run[1] : 0.f;
  if (CM) {
    // Merge of the cluster's splits: after every split finished its key range,
    // each CTA pushes the rows another rank owns, with its log-sum-exp, into
    // that rank's (now idle) K/V tile memory; one more barrier; then each
    // owner merges its rows locally in split order.
    cg::cluster_group cluster = cg::this_cluster();
    const int S = static_cast<int>(cluster.num_blocks());
    const int rank = static_cast<int>(cluster.block_rank());
    const int rows_per = (kTokTile + S - 1) / S;
    // [S][rows_per][kD] + [S][rows_per]: at most 55 rows (S <= 8), 28.4 KB, placed
    // at the start of the (idle) staging memory (48 KB or more; checked above)
    float* rPo = reinterpret_cast<float*>(smem);
    float* rLse = rPo + static_cast<size_t>(S) * rows_per * kD;  // [S][rows_per]
    cluster.sync();  // every split is done with its tiles
    {
      const int own0 = qr0 / rows_per, own1 = qr1 / rows_per;
      float* d0 = cluster.map_shared_rank(rPo, own0) + (static_cast<size_t>(rank) * rows_per + (qr0 - own0 * rows_per)) * kD;
      float* d1 = cluster.map_shared_rank(rPo, own1) + (static_cast<size_t>(rank) * rows_per + (qr1 - own1 * rows_per)) * kD;
#pragma unroll
      for (int n = 0; n < 16; ++n) {
        const int d = n * 8 + 2 * (lane & 3);
        *reinterpret_cast<float2*>(d0 + d) = make_float2(o_acc[n][0] * inv0, o_acc[n][1] * inv0);
        *reinterpret_cast<float2*>(d1 + d) = make_float2(o_acc[n][2] * inv1, o_acc[n][3] * inv1);
      }
      if ((lane & 3) == 0) {
        cluster.map_shared_rank(rLse, own0)[rank * rows_per + (qr0 - own0 * rows_per)] =
            l_run[0] > 0.f ? m_run[0] + log2f(l_run[0]) : -CUDART_INF_F;
        cluster.map_shared_rank(rLse, own1)[rank * rows_per + (qr1 - own1 * rows_per)] =
            l_run[1] > 0.f ? m_run[1] + log2f(l_run[1]) : -CUDART_INF_F;
      }
    }
    cluster.sync();  // all pushes landed
    const int q_lo = rank * rows_per;
    const int q_hi = min(p.n_q, q_lo + rows_per);
    for (int i = tid; i < (q_hi - q_lo) * (kD / 4); i += kThreads) {
      const int qq = i / (kD / 4);
      const int q = q_lo + qq;
      const int d = (i % (kD / 4)) * 4;
      float mmax = -CUDART_INF_F;
      for (int r = 0; r < S; ++r) mmax = fmaxf(mmax, rLse[r * rows_per + qq]);
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      float wsum = 0.f;
      if (mmax != -CUDART_INF_F) {
        for (int r = 0; r < S; ++r) {
          const float w = exp2f(rLse[r * rows_per + qq] - mmax);
          const float4 v = *reinterpret_cast<const float4*>(rPo + (static_cast<size_t>(r) * rows_per + qq) * kD + d);
          wsum += w;
          acc.x += w * v.x;
          acc.y += w * v.y;
          acc.z += w * v.z;
          acc.w += w * v.w;
        }
      }
      const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
      uint2 packed;
      packed.x = pack_half2(acc.x * inv, acc.y * inv);
      packed.y = pack_half2(acc.z * inv, acc.w * inv);
      *reinterpret_cast<uint2*>(p.out + (static_cast<size_t>(b) * p.n_q + q) * p.out_stride + h * kD + d) = packed;
      if (p.lse != nullptr && d == 0)
        p.lse[(static_cast<size_t>(b) * H + h) * p.n_q + q] =
            wsum > 0.f ? (mmax + log2f(wsum)) * 0.6931471805599453f : -CUDART_INF_F;
    }
    return;
  }
  if (p.n_splits == 1) {
    const bool v0 = qr0 < p.n_q;
    const bool v1 = qr1 < p.n_q;
    __half* out0 = p.out + (static_cast<size_t>(b) * p.n_q + qr0) * p.out_stride + h * kD;
    __half* out1 = p.out + (static_cast<size_t>(b) * p.n_q + qr1) * p.out_stride + h * kD;
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      const int d = n * 8 + 2 * (lane & 3);
      if (v0) *reinterpret_cast<uint32_t*>(out0 + d) = pack_half2(o_acc[n][0] * inv0, o_acc[n][1] * inv0);
      if (v1) *reinterpret_cast<uint32_t*>(out1 + d) = pack_half2(o_acc[n][2] * inv1, o_acc[n][3] * inv1);
    }
    if (p.lse != nullptr && (lane & 3) == 0) {
      const float ln2 = 0.6931471805599453f;
      if (v0) p.lse[(static_cast<size_t>(b) * H + h) * p.n_q + qr0] = (m_run[0] + log2f(l_run[0])) * ln2;
      if (v1) p.lse[(static_cast<size_t>(b) * H + h) * p.n_q + qr1] = (m_run[1] + log2f(l_run[1])) * ln2;
    }
  } else {
    float* po = p.part_o + part_base * kTokTile * kD;
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      const int d = n * 8 + 2 * (lane & 3);
      *reinterpret_cast<float2*>(po + static_cast<size_t>(qr0) * kD + d) =
          make_float2(o_acc[n][0] * inv0, o_acc[n][1] * inv0);
      *reinterpret_cast<float2*>(po + static_cast<size_t>(qr1) * kD + d) =
          make_float2(o_acc[n][2] * inv1, o_acc[n][3] * inv1);
    }
    if ((lane & 3) == 0) {
      p.part_lse[part_base * kTokTile + qr0] = m_run[0] + log2f(l_run[0]);
      p.part_lse[part_base * kTokTile + qr1] = m_run[1] + log2f(l_run[1]);
    }
  }
}

// Merge of the split partials: one warp per (head, vehicle, query), lane = 4 dims; the
// splits are added in split order.
__global__ void __launch_bounds__(256) attn_combine_kernel(const AttnArgs p) {
  const int h = blockIdx.x;
  const int b = blockIdx.y;
  const int qi = blockIdx.z * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int H = p.n_heads;
  const int S = p.n_splits;
  pdl_launch_dependents();
  pdl_wait();
  if (*reinterpret_cast<volatile int*>(p.status) != 0 || qi >= p.n_q) return;
  const size_t base = (static_cast<size_t>(b) * H + h) * S;
  float mmax = -CUDART_INF_F;
  for (int s = 0; s < S; ++s) mmax = fmaxf(mmax, p.part_lse[(base + s) * kTokTile + qi]);
  float wsum = 0.f;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  if (mmax != -CUDART_INF_F) {
    for (int s = 0; s < S; ++s) {
      const float w = exp2f(p.part_lse[(base + s) * kTokTile + qi] - mmax);
      const float4 v = *reinterpret_cast<const float4*>(p.part_o + ((base + s) * kTokTile + qi) * kD + lane * 4);
      wsum += w;
      acc.x += w * v.x;
      acc.y += w * v.y;
      acc.z += w * v.z;
      acc.w += w * v.w;
    }
  }
  const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
  uint2 pk;
  pk.x = pack_half2(acc.x * inv, acc.y * inv);
  pk.y = pack_half2(acc.z * inv, acc.w * inv);
  *reinterpret_cast<uint2*>(p.out + (static_cast<size_t>(b) * p.n_q + qi) * p.out_stride + h * kD + lane * 4) = pk;
  if (p.lse != nullptr && lane == 0)
    p.lse[(static_cast<size_t>(b) * H + h) * p.n_q + qi] =
        wsum > 0.f ? (mmax + log2f(wsum)) * 0.6931471805599453f : -CUDART_INF_F;
}

}  // namespace

size_t attention_workspace_bytes(int B, int n_heads, int n_splits) {
  if (n_splits <= kMaxClusterSplits) return 0;  // one split writes directly, up to 8 merge in a cluster
  const size_t parts = static_cast<size_t>(B) * n_heads * n_splits;
  return parts * kTokTile * kD * sizeof(float) + parts * kTokTile * sizeof(float);
}

int attention_launch_count(int n_splits) { return n_splits > kMaxClusterSplits ? 2 : 1; }

cudaError_t attention_set_attributes() {
  const void* fns[4] = {reinterpret_cast<const void*>(&attn_splitkv_kernel<__nv_bfloat16, false>),
                        reinterpret_cast<const void*>(&attn_splitkv_kernel<__nv_bfloat16, true>),
                        reinterpret_cast<const void*>(&attn_splitkv_kernel<float, false>),
                        reinterpret_cast<const void*>(&attn_splitkv_kernel<float, true>)};
  const size_t bytes[4] = {attn_smem_bytes<__nv_bfloat16>(), attn_smem_bytes<__nv_bfloat16>(),
                           attn_smem_bytes<float>(), attn_smem_bytes<float>()};
  for (int i = 0; i < 4; ++i) {
    cudaError_t e = cudaFuncSetAttribute(fns[i], cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes[i]));
    if (e != cudaSuccess) return e;
  }
  return attention_tc_set_attributes();
}

cudaError_t launch_attention(const AttnArgs& a_in, int B, int cache_dtype, cudaStream_t stream, bool pdl) {
  if (attention_tc_eligible(a_in, cache_dtype)) return launch_attention_tc(a_in, B, stream, pdl);
  AttnArgs a = a_in;
  void* kargs[] = {&a};
  const dim3 grid(a.n_splits, a.n_heads, B);
  const bool cm = a.n_splits > 1 && a.n_splits <= kMaxClusterSplits;
  const void* fn;
  size_t smem;
  if (cache_dtype == 1) {
    fn = cm ? reinterpret_cast<const void*>(&attn_splitkv_kernel<__nv_bfloat16, true>)
            : reinterpret_cast<const void*>(&attn_splitkv_kernel<__nv_bfloat16, false>);
    smem = attn_smem_bytes<__nv_bfloat16>();
  } else {
    fn = cm ? reinterpret_cast<const void*>(&attn_splitkv_kernel<float, true>)
            : reinterpret_cast<const void*>(&attn_splitkv_kernel<float, false>);
    smem = attn_smem_bytes<float>();
  }
  cudaError_t e = launch_ex(fn, grid, dim3(kThreads), smem, stream, pdl, kargs, 1, cm ? a.n_splits : 1);
  if (e != cudaSuccess || a.n_splits <= kMaxClusterSplits) return e;
  return launch_ex(reinterpret_cast<const void*>(&attn_combine_kernel), dim3(a.n_heads, B, (a.n_q + 7) / 8), dim3(256),
                   0, stream, pdl, kargs);
}

}  // namespace fsx
