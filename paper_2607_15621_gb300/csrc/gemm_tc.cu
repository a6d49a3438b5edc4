// Tensor-core (tcgen05 / TMEM) projection GEMMs of the expert layer (Sec. 3.1:
// W_q/W_k/W_v, W_o and the SwiGLU block) for batches of vehicles, where the
// token count M = 42 B makes them real dense contractions.
//
// D[128 weight rows, BN tokens] = W_tile[128, K] . A[BN tokens, K]^T, fp16
// operands, fp32 accumulation in tensor memory. The kernel is persistent: one
// CTA per SM walks the (weight tile, token block) tiles gridDim.x apart, and
// its warps specialise:
//   warp 0 (one lane): producer -- per 64-wide K step, the weight tile arrives
//     as one 16 KB bulk copy of a pre-swizzled image (packed at fsx_create in
//     the 128-byte swizzle layout the MMA reads), the token tile by a 2-D TMA
//     load with the same swizzle (rows past M read as zeros), through a
//     4-stage ring that runs on across tile boundaries;
//   warp 1 (one lane): issues tcgen05.mma (M=128, N=BN, K=16) x4 per stage,
//     releases each stage to the producer, and alternates between two
//     accumulators in tensor memory, so the MMAs of tile i+1 run while the
//     epilogue drains tile i;
//   warps 2-13: epilogue, three groups of 4 warps taking 32-token chunks in turn --
//     fp16 output and SwiGLU (gate rows 16j..16j+7 next to their up rows): the
//     chunk is read from TMEM in the 16x256b shape (mma accumulator fragments),
//     scaled, packed to fp16 (SwiGLU: each thread holds a gate value beside its
//     up value) and written transposed into a token-major staging tile by
//     stmatrix, then stored as 16-byte row pieces; the fp32 residual update
//     reads its 32 lanes in the 32x32b shape (each element owned by one thread)
//     and also emits each token's sum of x^2 over its 128 columns.
// Pair variant (opt-in for QKV at 256-token tiles and 2048 tokens or more): a cluster of two CTAs on an SM
// pair computes D[256 weight rows, 256 tokens] with tcgen05.mma.cta_group::2 (M = 256):
// each CTA stages its own 128-row weight tile and half of the 256 token rows (32 KB per
// stage instead of 48, so six stages fit instead of four), the even CTA issues the MMAs
// for both, and each CTA's tensor memory receives the accumulator of its own weight rows
// over all 256 tokens, so the epilogue is the single-CTA one. Both CTAs' copies complete
// on the even CTA's stage barriers; its commits arrive on both CTAs' barriers.
// RMSNorm-fused GEMMs (QKV, gate/up) take the fp16 copy of the residual stream
// as A, with the norm gain folded into the packed weights, and scale each
// token's result by 1/rms built from those per-128-column sums in a fixed
// order (so the norm costs no extra pass and stays deterministic).
#include <cuda.h>

#include "device_util.cuh"
#include "gemm_tc.h"
#include "tcgen05.cuh"

namespace fsx {

namespace {

constexpr int kEpiGroups = 3;         // epilogue groups of 4 warps (one per TMEM lane quadrant)
constexpr int kEpiThreads = kEpiGroups * 128;
constexpr int kTcThreads = 64 + kEpiThreads;  // producer warp, MMA warp, epilogue groups
constexpr int kTileN = 128;           // weight rows per tile (MMA M)
constexpr int kTileK = 64;            // K per stage (128 bytes of fp16: one swizzle span)
constexpr int kWTileBytes = kTileN * kTileK * 2;  // 16 KB
constexpr int kEpiChunk = 32;                     // tokens per epilogue round of one half
constexpr int kStgHalfBytes = 8192;               // fp16 staging of one group: 32 tokens x 128 columns (two TMA boxes)
constexpr int kSspBytes = ((kEpiGroups * 32 * 4 * 4 + 1023) / 1024) * 1024;  // x^2 partials [groups][32][4]

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_addr(dst)),
      "l"(map), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}

// TMA store of a (64 columns x 32 rows) box of the output from 128-byte swizzled shared memory
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(map),
               "r"(smem_addr(src)), "r"(x), "r"(y)
               : "memory");
}

// Copies of the pair variant: they land in this CTA's shared memory and complete on the
// barrier at cluster address `bar` (the even CTA's). A weight tile is one 16 KB box of
// the 3-D map [tiles][128 rows][64] over the packed images (no swizzle: the images are
// stored in the operand layout already).
__device__ __forceinline__ void tma_load_w_pair(void* dst, const CUtensorMap* map, int tile, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, {%2, "
      "%3, %4}], [%5];" ::"r"(smem_addr(dst)),
      "l"(map), "r"(0), "r"(0), "r"(tile), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2 [%0], [%1, {%2, "
      "%3}], [%4];" ::"r"(smem_addr(dst)),
      "l"(map), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ uint32_t cta0_addr(const void* local) {  // same offset in cluster CTA 0
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, 0;" : "=r"(r) : "r"(smem_addr(local)));
  return r;
}
// D (+)= A B^T over the CTA pair (M = 256: A rows from both CTAs, B rows split by N)
__device__ __forceinline__ void umma_f16_pair(uint32_t tmem_d, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                              uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// arrive on the barrier at this offset in the CTAs of `mask` once the pair MMAs issued so far completed
__device__ __forceinline__ void umma_commit_pair(uint64_t* bar, uint16_t mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
          smem_addr(bar)),
      "h"(mask)
      : "memory");
}
// Two 16-lane halves of the warp's TMEM lane quadrant, 32 columns each (16x256b shape, x4):
// thread t holds, for columns 8i .. 8i + 7, r[4i] = (lane t/4, column 8i + 2(t%4)), r[4i + 1] the
// next column, r[4i + 2] / r[4i + 3] the same columns of lane t/4 + 8 -- the mma.sync
// accumulator fragment, which stmatrix takes directly.
__device__ __forceinline__ void tmem_ld16x256_x4(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.16x256b.x4.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld2x16(uint32_t (&a)[16], uint32_t (&b)[16]) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;"
      : "+r"(a[0]), "+r"(a[1]), "+r"(a[2]), "+r"(a[3]), "+r"(a[4]), "+r"(a[5]), "+r"(a[6]), "+r"(a[7]), "+r"(a[8]),
        "+r"(a[9]), "+r"(a[10]), "+r"(a[11]), "+r"(a[12]), "+r"(a[13]), "+r"(a[14]), "+r"(a[15]), "+r"(b[0]),
        "+r"(b[1]), "+r"(b[2]), "+r"(b[3]), "+r"(b[4]), "+r"(b[5]), "+r"(b[6]), "+r"(b[7]), "+r"(b[8]), "+r"(b[9]),
        "+r"(b[10]), "+r"(b[11]), "+r"(b[12]), "+r"(b[13]), "+r"(b[14]), "+r"(b[15])
      :
      : "memory");
}
// four 8x8 fp16 matrices given as accumulator fragments, stored transposed: lanes 8i .. 8i + 7
// give the addresses of rows 0-7 of matrix i, and row j of the stored matrix is column j of
// the fragment's matrix (16 bytes)
__device__ __forceinline__ void stsm_x4_trans(uint32_t addr, uint32_t r0, uint32_t r1, uint32_t r2, uint32_t r3) {
  asm volatile("stmatrix.sync.aligned.m8n8.x4.trans.shared.b16 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(r0), "r"(r1),
               "r"(r2), "r"(r3)
               : "memory");
}

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// barrier among the 4 warps of epilogue group h (ids 1 .. kEpiGroups) / all epilogue warps
__device__ __forceinline__ void half_sync(int h) { asm volatile("bar.sync %0, 128;" ::"r"(1 + h) : "memory"); }
__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync %0, %1;" ::"n"(1 + kEpiGroups), "n"(kEpiThreads) : "memory"); }

template <int BN, bool PAIR = false>
__host__ __device__ constexpr int tc_stage_bytes() {  // the pair variant stages half of the token rows
  return kWTileBytes + (PAIR ? BN / 2 : BN) * kTileK * 2;
}

// Depth of the stage ring. A stage stays in flight for a round trip set by the L2 / HBM
// latency under load (copy issue, transfer, MMAs, release), so the ring takes as many
// stages as the shared memory holds: 4 of 48 KB for 256-token tiles, 5 of 34 KB for 144,
// 6 of 32 KB for 128, 8 of 22 KB for 48.
template <int BN, bool PAIR = false>
__host__ __device__ constexpr int tc_stages() {
  return PAIR ? 6 : (BN >= 256 ? 4 : (BN >= 144 ? 5 : (BN >= 128 ? 6 : 8)));
}

template <int BN>
__host__ __device__ constexpr int tc_rstd_bytes() {  // 1/rms of the tokens, double-buffered by tile parity
  return ((2 * BN * 4 + 1023) / 1024) * 1024;
}
// a 32-token chunk read of the 1/rms buffer may run past BN (last chunk of BN = 48)
static_assert(tc_rstd_bytes<48>() >= (2 * 48 + 32) * 4, "1/rms buffer too small for a 32-token read");
static_assert(kStgHalfBytes % 1024 == 0 && kSspBytes % 1024 == 0, "the stage ring must stay 1024-byte aligned");

template <int BN, bool PAIR = false>
__host__ __device__ constexpr int tc_smem_bytes() {
  return 1024 /* barriers, tmem address */ + tc_rstd_bytes<BN>() + kSspBytes + kEpiGroups * kStgHalfBytes +
         1024 /* alignment slack */ + tc_stages<BN, PAIR>() * tc_stage_bytes<BN, PAIR>();
}

static_assert(tc_smem_bytes<256>() <= 232448 && tc_smem_bytes<144>() <= 232448 && tc_smem_bytes<128>() <= 232448 &&
                  tc_smem_bytes<48>() <= 232448 && tc_smem_bytes<256, true>() <= 232448,
              "shared memory of a tile shape exceeds the per-block limit");
static_assert(2 * 8 * 8 + 2 * 2 * 8 + 8 <= 1024, "barriers of the deepest ring exceed the header");

template <int BN>
__host__ __device__ constexpr uint32_t tc_tmem_cols() {  // two accumulators, power of two >= 32
  return 2 * BN <= 32 ? 32 : (2 * BN <= 64 ? 64 : (2 * BN <= 128 ? 128 : (2 * BN <= 256 ? 256 : 512)));
}

template <int BN, int EPI, bool NORM, bool PAIR>
__global__ void __launch_bounds__(kTcThreads, 1) gemm_tc_kernel(const __grid_constant__ CUtensorMap map_a,
                                                               const __grid_constant__ CUtensorMap map_w,
                                                               const __grid_constant__ CUtensorMap map_y,
                                                               const TcGemmArgs p) {
  static_assert(!PAIR || (BN == 256 && EPI != kEpiResidual), "the pair variant runs 256-token store / SwiGLU tiles");
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  constexpr int kStages = tc_stages<BN, PAIR>();
  constexpr int kStageBytes = tc_stage_bytes<BN, PAIR>();
  // 1024-byte aligned stage area (the swizzle pattern repeats every 1024 bytes)
  unsigned char* base = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(base);
  uint64_t* empty = full + kStages;
  uint64_t* tmem_full = empty + kStages;   // [2] accumulator ready for the epilogue
  uint64_t* tmem_empty = tmem_full + 2;    // [2] accumulator drained (pair: by both CTAs' epilogues)
  uint64_t* mma_drain = tmem_empty + 2;    // pair: the last MMAs of the even CTA
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_drain + 1);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);  // a wait of this CTA timed out
  float* s_rstd = reinterpret_cast<float*>(base + 1024);                    // [2][BN]
  float* s_ssp = reinterpret_cast<float*>(base + 1024 + tc_rstd_bytes<BN>());  // [groups][32 tokens][4 quadrants]
  unsigned char* stg = base + 1024 + tc_rstd_bytes<BN>() + kSspBytes;        // [groups] fp16 staging
  unsigned char* stages = stg + kEpiGroups * kStgHalfBytes;

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int KT = p.K / kTileK;
  const int tiles_n = p.N / kTileN;
  const int n_tiles = tiles_n * ((p.M + BN - 1) / BN);
  const int KS = (EPI == kEpiResidual && p.k_splits > 1) ? p.k_splits : 1;
  uint32_t crank = 0;  // pair: this CTA's rank in the cluster (0 issues the MMAs)
  if (PAIR) asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(crank));
  // unit u: tile tile_of(u), K steps [kt0(u), kt1(u)). Pair units are (weight tile pair,
  // token block); the CTA of rank c takes the pair's weight tile 2 j + c.
  const int half_n = tiles_n / 2;
  const int n_units = PAIR ? n_tiles / 2 : n_tiles * KS;
  const int u_first = PAIR ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int u_step = PAIR ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);
  auto tile_of = [&](int u) {
    return PAIR ? (u / half_n) * tiles_n + (u % half_n) * 2 + static_cast<int>(crank) : u / KS;
  };
  auto kt0 = [&](int u) { return (u % KS) * KT / KS; };
  auto kt1 = [&](int u) { return (u % KS + 1) * KT / KS; };
  constexpr int kAbytes = (PAIR ? BN / 2 : BN) * kTileK * 2;
  constexpr uint32_t kTmemCols = tc_tmem_cols<BN>();
  // bounded wait that gives up at once after an earlier timeout of this CTA
  auto wait = [&](uint64_t* bar, uint32_t parity) {
    if (*abort) return;
    if (!mbar_wait(bar, parity, p.status)) *abort = 1;
  };

  pdl_launch_dependents();
  if (tid == 0) {
    *abort = 0;
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tmem_full + a, 1);
      mbar_init(tmem_empty + a, (PAIR ? 2 : 1) * 4 * kEpiGroups);  // one arrival per epilogue warp
    }
    mbar_init(mma_drain, 1);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0) {  // tensor memory for two accumulators of BN fp32 columns x 128 lanes
    if (PAIR) {  // allocated together by one warp of each CTA of the pair
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_slot)),
                   "r"(kTmemCols)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_slot)),
                   "r"(kTmemCols)
                   : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  if (PAIR) cluster_sync_all();  // both CTAs' barriers initialised before any copy or commit reaches them
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(tmem_slot);

  if (warp == 0) {
    // ---- producer (converged; lane 0 issues). Stage g of this CTA's stream runs
    // over its units in order and over each unit's K steps. Weights may stream
    // before the previous kernel finished, the token tiles only after it.
    auto w_src = [&](int u, int kt) {
      return p.w + (static_cast<size_t>(tile_of(u) % tiles_n) * KT + kt) * kWTileBytes;
    };
    // pair: the weight tile's index in the map over all packed tiles, the even CTA's
    // barrier of stage s, and the bytes both CTAs deliver to it
    auto w_tile = [&](int u, int kt) { return p.w_tile0 + (tile_of(u) % tiles_n) * KT + kt; };
    auto pair_bar = [&](int s) { return cta0_addr(full + s); };
    constexpr uint32_t kPairTx = 2u * (kWTileBytes + kAbytes);
    if (lane == 0) {
      int g = 0;
      for (int u = u_first; u < n_units && g < kStages; u += u_step)
        for (int kt = kt0(u); kt < kt1(u) && g < kStages; ++kt, ++g) {
          if (PAIR) {
            if (crank == 0) mbar_arrive_expect_tx(full + g, kPairTx);
            tma_load_w_pair(stages + g * kStageBytes, &map_w, w_tile(u, kt), pair_bar(g));
          } else {
            mbar_arrive_expect_tx(full + g, kWTileBytes + kAbytes);
            bulk_g2s(stages + g * kStageBytes, w_src(u, kt), kWTileBytes, full + g);
          }
        }
    }
    __syncwarp();
    pdl_wait();
    int total = 0;
    for (int u = u_first; u < n_units; u += u_step) {
      const int m_tile = tile_of(u) / tiles_n;
      for (int kt = kt0(u); kt < kt1(u); ++kt, ++total) {
        const int g = total;
        const int s = g % kStages;
        unsigned char* st = stages + s * kStageBytes;
        if (g >= kStages) wait(empty + s, static_cast<uint32_t>(((g / kStages) - 1) & 1));
        if (PAIR) {  // after a timeout of this CTA no further copy is issued
          if (lane == 0 && *abort == 0) {
            if (g >= kStages) {
              if (crank == 0) mbar_arrive_expect_tx(full + s, kPairTx);
              tma_load_w_pair(st, &map_w, w_tile(u, kt), pair_bar(s));
            }
            tma_load_2d_pair(st + kWTileBytes, &map_a, kt * kTileK, m_tile * BN + static_cast<int>(crank) * (BN / 2),
                             pair_bar(s));
          }
        } else if (lane == 0) {
          if (g >= kStages) {
            mbar_arrive_expect_tx(full + s, kWTileBytes + kAbytes);
            bulk_g2s(st, w_src(u, kt), kWTileBytes, full + s);
          }
          tma_load_2d(st + kWTileBytes, &map_a, kt * kTileK, m_tile * BN, full + s);
        }
        __syncwarp();
      }
    }
    // after a timeout the MMA warp may have skipped its waits: let the copies still in
    // flight land (bounded) before the shared memory is released (the pair variant
    // waits at its exit instead)
    if (!PAIR && *abort && lane == 0)
      for (int g = total - kStages; g < total; ++g) {
        if (g < 0) continue;
        const unsigned long long t0 = global_timer_ns();
        uint32_t done = 0;
        while (!done && global_timer_ns() - t0 < 100000000ull)
          asm volatile(
              "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
              : "=r"(done)
              : "r"(smem_addr(full + g % kStages)), "r"(static_cast<uint32_t>((g / kStages) & 1))
              : "memory");
      }
    __syncwarp();
  } else if (warp == 1 && PAIR && crank != 0) {
    // the odd CTA of a pair issues no MMAs
  } else if (warp == 1) {
    // ---- MMA issuer (converged; lane 0 issues)
    pdl_wait();
    constexpr uint32_t idesc = idesc_f16(PAIR ? 2 * kTileN : kTileN, BN);
    int g = 0;
    int i = 0;
    for (int u = u_first; u < n_units; u += u_step, ++i) {
      const int acc = i & 1;
      if (i >= 2) {
        const uint32_t par = static_cast<uint32_t>(((i >> 1) - 1) & 1);
        if (PAIR) {  // drained by the epilogues of both CTAs
          if (*abort == 0 && !mbar_wait_cluster(tmem_empty + acc, par, p.status)) *abort = 1;
        } else {
          wait(tmem_empty + acc, par);
        }
      }
      tc_fence_after();
      const uint32_t d = tmem + static_cast<uint32_t>(acc * BN);
      const int k_first = kt0(u);
      for (int kt = k_first; kt < kt1(u); ++kt, ++g) {
        const int s = g % kStages;
        wait(full + s, static_cast<uint32_t>((g / kStages) & 1));
        tc_fence_after();
        if (lane == 0 && !(PAIR && *abort)) {
          const uint32_t a_base = smem_addr(stages + s * kStageBytes);
          const uint32_t b_base = a_base + kWTileBytes;
#pragma unroll
          for (int k = 0; k < kTileK / 16; ++k) {
            if (PAIR)
              umma_f16_pair(d, sw128_desc(a_base + k * 32), sw128_desc(b_base + k * 32), idesc,
                            (kt > k_first || k > 0) ? 1u : 0u);
            else
              umma_f16(d, sw128_desc(a_base + k * 32), sw128_desc(b_base + k * 32), idesc,
                       (kt > k_first || k > 0) ? 1u : 0u);
          }
          if (PAIR)
            umma_commit_pair(empty + s, 3);  // both CTAs' producers may refill the stage
          else
            umma_commit(empty + s);
        }
        __syncwarp();
      }
      if (lane == 0 && !(PAIR && *abort)) {
        if (PAIR)
          umma_commit_pair(tmem_full + acc, 3);
        else
          umma_commit(tmem_full + acc);
      }
      __syncwarp();
    }
    if (PAIR) {  // every MMA of the pair done before either CTA frees its tensor memory
      if (lane == 0) umma_commit_pair(mma_drain, 1);
      __syncwarp();
      mbar_wait(mma_drain, 0u, p.status);
    }
  } else {
    // ---- epilogue: groups of 4 warps (warps 2-5, 6-9, ...) take the 32-token chunks
    // of a tile in turn; in each group TMEM lane quadrant q = warp % 4 holds weight
    // rows 32q..32q+31 (this thread: row 32q + lane)
    pdl_wait();  // the residual stream written by the previous kernel is read below
    const int etid = tid - 64;
    const int half = etid >> 7;  // epilogue group
    const int htid = etid & 127;
    const int q = warp & 3;
    const int row = q * 32 + lane;
    __half* tH = reinterpret_cast<__half*>(stg + half * kStgHalfBytes);
    float* ssp = s_ssp + half * kEpiChunk * 4;
    // x[m, n0 + row] += D[row, m] for the chunk's tokens: lanes hold consecutive columns,
    // so every access of the warp is one contiguous 128-byte row piece; also the
    // tokens' sums of x^2 over the tile's 128 columns
    auto residual_chunk = [&](int tn_, int m0, int c0, int nc, uint32_t (&r)[32]) {
      const int n0 = tn_ * kTileN;
      const int n_ok = min(nc, p.M - (m0 + c0));  // valid tokens of the chunk
      float* px = p.xo + static_cast<size_t>(m0 + c0) * p.ldxo + n0 + row;
      __half* ph = p.xo16 + static_cast<size_t>(m0 + c0) * p.ldxo + n0 + row;
      float x[32];
#pragma unroll
      for (int j = 0; j < 32; ++j)  // every load in flight before the first store
        x[j] = j < n_ok ? __ldcg(px + static_cast<size_t>(j) * p.ldxo) : 0.f;
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        x[j] += __uint_as_float(r[j]);
        if (j < n_ok) {
          px[static_cast<size_t>(j) * p.ldxo] = x[j];
          ph[static_cast<size_t>(j) * p.ldxo] = __float2half_rn(x[j]);
        }
        x[j] = j < n_ok ? x[j] * x[j] : 0.f;
      }
      // 32 tokens x 32 lanes of x^2 -> lane l holds this quadrant's sum for token l
#pragma unroll
      for (int sh = 16; sh > 0; sh >>= 1) {
        const bool upper = (lane & sh) != 0;
#pragma unroll
        for (int j = 0; j < sh; ++j) {
          const float send = upper ? x[j] : x[j + sh];
          const float keep = upper ? x[j + sh] : x[j];
          x[j] = keep + __shfl_xor_sync(0xffffffffu, send, sh);
        }
      }
      ssp[lane * 4 + q] = x[0];
      half_sync(half);
      if (htid < nc && p.ss_out != nullptr && m0 + c0 + htid < p.M)  // fixed quadrant order
        p.ss_out[static_cast<size_t>(tn_) * p.ss_stride + m0 + c0 + htid] =
            ((ssp[htid * 4 + 0] + ssp[htid * 4 + 1]) + ssp[htid * 4 + 2]) + ssp[htid * 4 + 3];
      half_sync(half);
    };
    int i = 0;
    for (int u = u_first; u < n_units; u += u_step, ++i) {
      const int acc = i & 1;
      const int tile = tile_of(u);
      const int split = u % KS;
      const int t_n = tile % tiles_n;
      const int n0 = t_n * kTileN;
      const int m0 = (tile / tiles_n) * BN;
      float* rstd = s_rstd + acc * BN;
      if (NORM) {  // 1/rms of the tile's tokens from the per-128-column partial sums of x^2
        for (int tt = etid; tt < BN; tt += kEpiThreads) {
          float ss = 0.f;
          if (m0 + tt < p.M)
            for (int j = 0; j < p.n_ss; ++j) ss += __ldcg(p.ss_in + static_cast<size_t>(j) * p.ss_stride + m0 + tt);
          rstd[tt] = rsqrtf(ss / static_cast<float>(p.K) + 1e-6f);
        }
      }
      wait(tmem_full + acc, static_cast<uint32_t>((i >> 1) & 1));
      tc_fence_after();
      epi_sync();  // 1/rms visible to both halves; both halves are past the previous tile
      const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN);
      for (int c0 = half * kEpiChunk; c0 < BN; c0 += kEpiGroups * kEpiChunk) {
        const int nc = BN - c0 < kEpiChunk ? BN - c0 : kEpiChunk;  // 16 for the last chunk of BN = 48
        __syncwarp();  // tcgen05.ld.sync.aligned needs the whole warp converged
        if (EPI == kEpiResidual) {
          uint32_t r[32];
          if (nc == kEpiChunk) {
            tmem_ld32_issue(taddr + static_cast<uint32_t>(c0), r);
            tmem_wait_ld32(r);
          } else {
            float v16[16];
            tmem_ld16(taddr + static_cast<uint32_t>(c0), v16);
#pragma unroll
            for (int j = 0; j < 16; ++j) r[j] = __float_as_uint(v16[j]);
#pragma unroll
            for (int j = 16; j < 32; ++j) r[j] = 0u;
          }
          if (KS == 1) {
            residual_chunk(t_n, m0, c0, nc, r);
          } else {  // this split's partial -> workspace ([tile][split][token][128 columns])
            float* pp = p.part + (static_cast<size_t>(tile * KS + split) * BN + c0) * kTileN + row;
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (j < nc) pp[static_cast<size_t>(j) * kTileN] = __uint_as_float(r[j]);
          }
        } else {
          // the chunk as accumulator fragments: ra = lanes 32q .. 32q + 15 of the quadrant
          // (weight rows), rb = lanes 32q + 16 .. 32q + 31; 32 token columns each (a short
          // last chunk of BN = 48 reads columns that are never stored)
          uint32_t ra[16], rb[16];
          tmem_ld16x256_x4(taddr + static_cast<uint32_t>(c0), ra);
          tmem_ld16x256_x4(taddr + (16u << 16) + static_cast<uint32_t>(c0), rb);
          tmem_wait_ld2x16(ra, rb);
          const int fq = lane & 3;  // fragment column pair: tokens 8i + 2 fq, 8i + 2 fq + 1
          float2 rs[4];             // their 1/rms (the 1/rms buffer has room past BN)
#pragma unroll
          for (int i = 0; i < 4; ++i)
            rs[i] = NORM ? *reinterpret_cast<const float2*>(rstd + c0 + 8 * i + 2 * fq) : make_float2(1.f, 1.f);
          auto val = [&](int hh, int k) {  // element k of the fragment registers of half hh
            return __uint_as_float(hh == 0 ? ra[k] : rb[k]);
          };
          // The chunk's fp16 outputs, 8x8 blocks as fragments: store -- weight rows
          // 32q + 8nb .. (nb = 2hh + {0, 1}), tokens 8i ..; SwiGLU -- packed rows 16b .. 16b + 7
          // are gate rows and 16b + 8 .. 16b + 15 their up rows, so a thread holds each gate
          // value (fragment row g) beside its up value (row g + 8): output columns
          // 8 (2q + hh) + g, tokens 8i + 2 fq (+1).
          constexpr int kNF = EPI == kEpiStore ? 16 : 8;
          uint32_t f[kNF];
#pragma unroll
          for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              const float a0 = val(hh, 4 * i) * rs[i].x, a1 = val(hh, 4 * i + 1) * rs[i].y;
              const float a2 = val(hh, 4 * i + 2) * rs[i].x, a3 = val(hh, 4 * i + 3) * rs[i].y;
              if (EPI == kEpiStore) {
                f[4 * i + 2 * hh] = pack_half2(a0, a1);
                f[4 * i + 2 * hh + 1] = pack_half2(a2, a3);
              } else {
                f[2 * i + hh] =
                    pack_half2(__fdividef(a0, 1.f + __expf(-a0)) * a2, __fdividef(a1, 1.f + __expf(-a1)) * a3);
              }
            }
          // the group's staging tile is free once its previous TMA store has read it
          if (htid == 0) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
          half_sync(half);
          // stmatrix (transposed) into the staging tile in the layout of the output TMA box:
          // 64 columns x 32 tokens per 4 KB box, token row r at 128 r, 16-byte unit u at
          // u ^ (r mod 8) (the 128-byte swizzle; the 8 rows of a matrix hit 8 bank groups)
          const uint32_t sbase = smem_addr(tH);
          const int tr = lane & 7;  // row of the matrix this lane addresses
          if (EPI == kEpiStore) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int tok = 8 * i + tr;
              const int col = 32 * q + 8 * (lane >> 3);
              const uint32_t a = sbase + (col >> 6) * 4096 + tok * 128 + ((((col & 63) >> 3) ^ (tok & 7)) << 4);
              stsm_x4_trans(a, f[4 * i], f[4 * i + 1], f[4 * i + 2], f[4 * i + 3]);
            }
          } else {
#pragma unroll
            for (int ip = 0; ip < 2; ++ip) {
              const int mi = lane >> 3;  // matrix mi: half mi & 1, token block 2 ip + mi / 2
              const int tok = 8 * (2 * ip + (mi >> 1)) + tr;
              const int u = 2 * q + (mi & 1);
              stsm_x4_trans(sbase + tok * 128 + ((u ^ (tok & 7)) << 4), f[4 * ip], f[4 * ip + 1], f[4 * ip + 2],
                            f[4 * ip + 3]);
            }
          }
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // staging -> TMA store
          half_sync(half);
          // one thread stores the chunk's token rows (rows past M are clipped by the map)
          if (htid == 0 && m0 + c0 < p.M) {
            if (EPI == kEpiStore) {
              tma_store_2d(&map_y, tH, n0, m0 + c0);
              tma_store_2d(&map_y, reinterpret_cast<const unsigned char*>(tH) + 4096, n0 + 64, m0 + c0);
            } else {
              tma_store_2d(&map_y, tH, n0 / 2, m0 + c0);
            }
            asm volatile("cp.async.bulk.commit_group;" ::: "memory");
          }
        }
      }
      // accumulator drained: hand it back to the MMA warp (pair: the even CTA's)
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (PAIR)
          asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cta0_addr(tmem_empty + acc))
                       : "memory");
        else
          mbar_arrive(tmem_empty + acc);
      }
      if (EPI == kEpiResidual && KS > 1) {
        // every split of the tile waits until all KS partials are written (the grid holds
        // at most one CTA per SM and never more CTAs than SMs, so all splits are resident),
        // then adds the partials of its own slice of tokens in split order
        __threadfence();
        epi_sync();
        if (etid == 0 && *abort == 0) {
          atomicAdd(p.tile_count + tile, 1);
          const unsigned long long t0 = global_timer_ns();
          for (uint32_t it = 0;; ++it) {
            int v;
            asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p.tile_count + tile) : "memory");
            if (v >= KS) break;
            if ((it & 63u) == 63u && global_timer_ns() - t0 > kWaitLimitNs) {
              set_status(p.status, kStatusTimeout);
              *abort = 1;
              break;
            }
          }
        }
        epi_sync();
        __threadfence();
        const int tk_lo = split * BN / KS;
        const int tk_hi = (split + 1) * BN / KS;
        // warp ew takes tokens tk_lo + ew, + 12, ...; lane = 4-column group of the tile's
        // 128 columns; 4 tokens' loads in flight at once
        const int ew = etid >> 5;
        constexpr int kEW = kEpiThreads / 32;
        for (int tk0 = tk_lo + ew; tk0 < tk_hi; tk0 += 4 * kEW) {
          float4 acc4[4];
#pragma unroll
          for (int bb = 0; bb < 4; ++bb) acc4[bb] = make_float4(0.f, 0.f, 0.f, 0.f);
          for (int sp = 0; sp < KS; ++sp) {
            const float* pp = p.part + (static_cast<size_t>(tile * KS + sp) * BN) * kTileN + lane * 4;
            float4 w4[4];
#pragma unroll
            for (int bb = 0; bb < 4; ++bb) {
              const int tk = tk0 + bb * kEW;
              w4[bb] = tk < tk_hi ? __ldcg(reinterpret_cast<const float4*>(pp + static_cast<size_t>(tk) * kTileN))
                                  : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int bb = 0; bb < 4; ++bb) {
              acc4[bb].x += w4[bb].x;
              acc4[bb].y += w4[bb].y;
              acc4[bb].z += w4[bb].z;
              acc4[bb].w += w4[bb].w;
            }
          }
#pragma unroll
          for (int bb = 0; bb < 4; ++bb) {
            const int tk = tk0 + bb * kEW;
            const int m = m0 + tk;
            float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
            const size_t idx = static_cast<size_t>(m) * p.ldxo + n0 + lane * 4;
            if (tk < tk_hi && m < p.M) {
              const float4 x0 = __ldcg(reinterpret_cast<const float4*>(p.xo + idx));
              x = make_float4(x0.x + acc4[bb].x, x0.y + acc4[bb].y, x0.z + acc4[bb].z, x0.w + acc4[bb].w);
              *reinterpret_cast<float4*>(p.xo + idx) = x;
              uint2 pk;
              pk.x = pack_half2(x.x, x.y);
              pk.y = pack_half2(x.z, x.w);
              *reinterpret_cast<uint2*>(p.xo16 + idx) = pk;
            }
            const float ss = warp_sum(x.x * x.x + x.y * x.y + x.z * x.z + x.w * x.w);
            if (lane == 0 && tk < tk_hi && m < p.M && p.ss_out != nullptr)
              p.ss_out[static_cast<size_t>(t_n) * p.ss_stride + m] = ss;
          }
        }
        // departures: the last split to leave resets the counter for the next launch
        epi_sync();
        if (etid == 0 && atomicAdd(p.tile_count + tile, 1) == 2 * KS - 1) p.tile_count[tile] = 0;
      }
    }
    // the output stores of this group complete before the CTA leaves
    if (EPI != kEpiResidual && htid == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  if (PAIR) {
    // after a timeout, copies already issued (which may complete on the other CTA's
    // barriers) land within microseconds: give them 1 ms, then leave together
    if (tid == 0 && *abort) {
      const unsigned long long t0 = global_timer_ns();
      while (global_timer_ns() - t0 < 1000000ull) {
      }
    }
    cluster_sync_all();
    tc_fence_after();
    if (warp == 0)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  } else if (warp == 0) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

template <int BN, int EPI, bool NORM, bool PAIR>
const void* tc_fn() {
  return reinterpret_cast<const void*>(&gemm_tc_kernel<BN, EPI, NORM, PAIR>);
}

const void* tc_select(int bn, int epi, bool norm, bool pair, size_t* smem) {
#define FSX_TC(BN_, EPI_, NORM_)                                 \
  if (bn == BN_ && epi == EPI_ && norm == NORM_ && !pair) {      \
    *smem = tc_smem_bytes<BN_>();                                 \
    return tc_fn<BN_, EPI_, NORM_, false>();                      \
  }
#define FSX_TC_PAIR(BN_, EPI_, NORM_)                            \
  if (bn == BN_ && epi == EPI_ && norm == NORM_ && pair) {       \
    *smem = tc_smem_bytes<BN_, true>();                           \
    return tc_fn<BN_, EPI_, NORM_, true>();                       \
  }
  FSX_TC(48, kEpiStore, true)
  FSX_TC(48, kEpiStore, false)
  FSX_TC(48, kEpiSwiglu, true)
  FSX_TC(48, kEpiResidual, false)
  FSX_TC(128, kEpiStore, true)
  FSX_TC(128, kEpiSwiglu, true)
  FSX_TC(128, kEpiResidual, false)
  FSX_TC(144, kEpiResidual, false)
  FSX_TC(256, kEpiStore, true)
  FSX_TC(256, kEpiSwiglu, true)
  FSX_TC(256, kEpiResidual, false)
  FSX_TC_PAIR(256, kEpiStore, true)
#undef FSX_TC
#undef FSX_TC_PAIR
  return nullptr;
}

int g_pair_clusters = 0;  // co-resident CTA pairs of the pair variant (0: not available)

}  // namespace

cudaError_t gemm_tc_set_attributes() {
  const int bns[4] = {48, 128, 144, 256};
  const int epis[3] = {kEpiStore, kEpiSwiglu, kEpiResidual};
  for (int pair = 0; pair < 2; ++pair)
    for (int bn : bns)
      for (int epi : epis)
        for (int norm = 0; norm < 2; ++norm) {
          size_t smem = 0;
          const void* fn = tc_select(bn, epi, norm != 0, pair != 0, &smem);
          if (!fn) continue;
          cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
          if (e != cudaSuccess) return e;
        }
  // how many CTA pairs of the pair variant fit at once (one CTA per SM)
  size_t smem = 0;
  const void* fn = tc_select(256, kEpiStore, true, true, &smem);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2);
  cfg.blockDim = dim3(kTcThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = 2;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) {
    (void)cudaGetLastError();
    n = 0;
  }
  g_pair_clusters = n;
  return cudaSuccess;
}

int gemm_tc_pair_clusters() { return g_pair_clusters; }

int gemm_tc_k_splits(int tiles, int KT, int sm_count) {
  if (tiles <= 0 || tiles >= sm_count) return 1;
  int ks = sm_count / tiles;                // all units in one wave
  const int max_ks = KT / 4;                // at least 4 K steps (16 MMAs) per unit
  if (ks > max_ks) ks = max_ks;
  return ks < 1 ? 1 : ks;
}

// tiles x splits <= sm_count whenever splits > 1, and a partial tile is at most 128 x 256 fp32
size_t gemm_tc_part_bytes(int sm_count) { return static_cast<size_t>(sm_count) * kTileN * 256 * sizeof(float); }

cudaError_t launch_gemm_tc(const CUtensorMap& map_a, const TcGemmArgs& args, int bn, int epi, bool norm,
                           cudaStream_t stream, bool pdl, const CUtensorMap* map_w) {
  const bool pair = map_w != nullptr;
  size_t smem = 0;
  const void* fn = tc_select(bn, epi, norm, pair, &smem);
  if (!fn || args.N % kTileN != 0 || args.K % kTileK != 0) return cudaErrorInvalidValue;
  if (pair && ((args.N / kTileN) % 2 != 0 || args.k_splits > 1 || g_pair_clusters <= 0)) return cudaErrorInvalidValue;
  static int sm_count = 0;
  if (sm_count == 0) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sm_count, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess || sm_count <= 0) return e != cudaSuccess ? e : cudaErrorInvalidValue;
  }
  CUtensorMap map = map_a;
  CUtensorMap mapw{};
  if (pair) mapw = *map_w;
  // the store and SwiGLU epilogues write their output rows by TMA: a map over y[M, cols]
  // (row stride ldy) with 64-column x 32-token boxes in the 128-byte swizzle
  CUtensorMap mapy{};
  if (epi != kEpiResidual) {
    const int cols = epi == kEpiStore ? args.N : args.N / 2;
    if (args.y == nullptr || args.M <= 0 || (reinterpret_cast<uintptr_t>(args.y) & 15) != 0 || (args.ldy * 2) % 16 != 0 ||
        cols % 64 != 0 || args.ldy < cols || !encode_out_map(&mapy, args.y, static_cast<uint64_t>(args.M),
                                                             static_cast<uint64_t>(cols), static_cast<uint64_t>(args.ldy)))
      return cudaErrorInvalidValue;
  }
  TcGemmArgs a = args;
  void* kargs[] = {&map, &mapw, &mapy, &a};
  if (a.k_splits > 1 && (epi != kEpiResidual || a.part == nullptr || a.tile_count == nullptr)) return cudaErrorInvalidValue;
  const int units = (args.N / kTileN) * ((args.M + bn - 1) / bn) * (a.k_splits > 1 ? a.k_splits : 1);
  if (pair) {  // one cluster of two CTAs per pair unit, at most as many as are co-resident
    const int pairs = units / 2;
    const int clusters = pairs < g_pair_clusters ? pairs : g_pair_clusters;
    return launch_ex(fn, dim3(static_cast<unsigned>(2 * clusters)), dim3(kTcThreads), smem, stream, pdl, kargs, 1, 2);
  }
  const dim3 grid(static_cast<unsigned>(units < sm_count ? units : sm_count));
  return launch_ex(fn, grid, dim3(kTcThreads), smem, stream, pdl, kargs);
}

// Weight tile (n_tile, k_tile) as the shared-memory image the MMA reads:
// row r of the 128-row tile, 16-byte chunk c of its 128-byte K slice goes to
// (r / 8) * 1024 + (r % 8) * 128 + ((c ^ (r % 8)) * 16).
void pack_tc_tile(const float* const* rows, const float* col_scale, int k0, __half* out) {
  unsigned char* o = reinterpret_cast<unsigned char*>(out);
  for (int r = 0; r < kTileN; ++r) {
    const float* src = rows[r];
    for (int c = 0; c < 8; ++c) {
      __half* dst = reinterpret_cast<__half*>(o + (r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) * 16));
      for (int e = 0; e < 8; ++e) {
        const int k = k0 + c * 8 + e;
        dst[e] = __float2half_rn(src[k] * (col_scale ? col_scale[k] : 1.f));
      }
    }
  }
}

}  // namespace fsx

namespace fsx {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void* sym = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &sym, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || sym == nullptr)
      return nullptr;
    fn = reinterpret_cast<EncodeTiledFn>(sym);
  }
  return fn;
}

bool encode_act_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  const EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kTileK), box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_out_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t ld) {
  const EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {ld * 2};
  const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(kEpiChunk)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_weight_map(CUtensorMap* map, const void* base, uint64_t n_tiles) {
  const EncodeTiledFn fn = encode_fn();
  if (fn == nullptr || n_tiles == 0 || n_tiles > 0x7fffffffull) return false;
  const cuuint64_t dims[3] = {static_cast<cuuint64_t>(kTileK), static_cast<cuuint64_t>(kTileN), n_tiles};
  const cuuint64_t strides[2] = {static_cast<cuuint64_t>(kTileK) * 2, static_cast<cuuint64_t>(kWTileBytes)};
  const cuuint32_t box[3] = {static_cast<cuuint32_t>(kTileK), static_cast<cuuint32_t>(kTileN), 1};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_cache_map(CUtensorMap* map, const void* base, uint64_t rows, uint32_t n_heads) {
  const EncodeTiledFn fn = encode_fn();
  if (fn == nullptr || rows == 0 || n_heads == 0) return false;
  const cuuint64_t dims[3] = {128, n_heads, rows};
  const cuuint64_t strides[2] = {256, static_cast<cuuint64_t>(n_heads) * 256};
  const cuuint32_t box[3] = {64, 1, 64};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace fsx
