// Persistent single-vehicle tick: the whole expert forward (Sec. 3.1, Eq. 1)
// for one vehicle in ONE kernel launch, built for the latency of a B = 1 tick.
//
// Layout of the work: the grid is one thread-block cluster of 4 CTAs per
// attention head (H clusters, 4H CTAs, one CTA per SM, all co-resident).
// Every layer runs two phases separated by device-wide counters:
//   phase A (every cluster = one head h):
//     each CTA reads its 128 columns of x, converts them to fp16 and sends them
//     with the per-token partial sums of x^2 to the whole cluster; four warps
//     each run the tensor-core MMAs (tcgen05, accumulators in tensor memory) of
//     one K quarter as soon as that quarter has arrived, for the CTA's 96 rows
//     of [W_q; W_k; W_v] of head h (32 q, 32 k, 32 v dims; the RMSNorm gain is
//     folded into the weights and 1/rms is applied to the accumulator sum) ->
//     q goes to all 4 CTAs, k_ae and v_ae to the CTA that attends over the own
//     keys -> Eq. 1 over a quarter of [K_vlm ; K_ae] per CTA (cache rows staged
//     three 64-key chunks deep in the shared memory the QKV operands used) ->
//     the 4 fp32 split results merged (log-sum-exp weights), each CTA merging
//     12 rows and sending them to the others -> the CTA's 128 output columns of
//     o_h W_o^T (tcgen05) added into the next residual state with vector atomics
//     (cluster 0 also adds the residual itself).
//   phase B (clusters 0 .. F/64-1; cluster c owns SwiGLU columns 64c..64c+63):
//     each CTA reads only its 128 columns of x, converts them to fp16 and starts
//     the cluster's 128 gate/up rows over this K quarter at once, while the
//     per-token partial sums of x^2 go to the cluster -> the partials are
//     reduce-scattered so that each CTA sums its 16 gate + 16 up rows, scales
//     them by 1/rms and forms its 16 SwiGLU columns -> h sent to all 4 CTAs ->
//     the CTA's 128 output columns of h W_d^T (tcgen05) added into the next
//     residual state.
// The residual stream rotates through three fp32 buffers: a phase reads one,
// accumulates into the next (zeroed one phase earlier) and zeroes the third.
//
// Exchanges inside a cluster never use a cluster-wide barrier: a CTA writes
// into its partners' shared memory with st.async stores that complete on the
// partner's mbarrier (transaction bytes), and the partner waits on that
// barrier alone. Each exchange barrier completes once per layer; it is re-armed
// with the next layer's byte count right after its wait, which always precedes
// the device-wide counter the senders must pass before sending again.
//
// Weights never wait for activations: each CTA's weights are packed in the
// order it consumes them, as the swizzled K-major images the tensor core reads
// (128-byte swizzle, one 64-wide K slice per image), and streamed by bulk
// copies through a 6-slot ring of 16 KB that is refilled as soon as a GEMM has
// finished with its slots (slots 2-5 only once the attention has finished
// staging cache rows in them), so the HBM stream runs ahead across phases and
// layers. A layer takes 12 ring positions (6 of QKV, 2 of W_o, 2 of gate/up,
// 1 of W_d and one empty position; CTAs without SwiGLU work leave positions
// 8-11 empty), so the QKV images of every layer start at slot 0. The MMAs run
// with M = 128: the 96-row QKV images are padded with whatever follows them in
// shared memory, and the accumulator rows that produces are never read. Every
// GEMM is issued by four warps into four accumulators that the epilogue adds:
// one issuing thread pays a fixed cost per MMA that four issuers overlap.
#include <cooperative_groups.h>
#include <math_constants.h>

#include "device_util.cuh"
#include "kernels.h"
#include "persistent.h"
#include "tcgen05.cuh"

namespace cg = cooperative_groups;

namespace fsx {

namespace {

constexpr int kThr = kPersistThreads;  // 256 = 8 warps
constexpr int kCl = kPersistCluster;   // 4 CTAs per cluster
constexpr int kSlotBytes = kPersistChunk;
constexpr int kSlots = kPersistSlots;
constexpr int kLayerChunks = 2 * kSlots;      // ring positions per layer, empty ones included
constexpr int kD = kHeadDim;           // 128
constexpr int kKeyTile = 32;           // keys per staged attention tile
constexpr int kQS = kD + 8;            // fp16 row stride of q / own k / own v (halves)
constexpr int kDS = 128 + 4;           // fp32 row stride of the output transpose buffer
constexpr int kRowsPerRank = kTokTile / kCl;  // 12
constexpr int kQkvAtom = 3 * 32 * 128;        // one 64-wide K slice of the CTA's 96 QKV rows (12 KB)
constexpr int kActAtom = kTokTile * 128;      // one K slice of the 48 token rows (6 KB)
constexpr int kNAcc = 4;                      // accumulators: one per MMA-issuing warp
constexpr uint32_t kAccCols = 64;             // tensor-memory columns per accumulator (48 used)
constexpr uint32_t kTmemCols = kNAcc * kAccCols;
constexpr uint32_t kIdesc = idesc_f16(128, kTokTile);
constexpr int kRecvBytes = kRowsPerRank * kD * 4;  // merge partials one CTA sends another (fp32)
constexpr int kRsBytes = 32 * kTokTile * 4;        // gate/up partials one CTA sends another (fp32)
static_assert(kRecvBytes == kRsBytes, "the merge and the gate/up reduce-scatter share the receive buffer");

struct Smem {
  // byte offsets from the 1024-byte aligned base of the dynamic shared memory
  int bars, gss, rstd, ring, act, qbuf, ownk, ownv, tile, recv, recv_lse, total;
};

__host__ __device__ inline Smem smem_layout(int d) {
  Smem s{};
  s.bars = 0;                                  // mbarriers, TMEM address, abort flag
  s.gss = 512;                                 // [4 ranks][48] fp32 partial sums of x^2
  s.rstd = 512 + kCl * kTokTile * 4;           // [48] fp32 1 / rms per token
  int o = 2048;
  s.ring = o;      o += kSlots * kSlotBytes;   // also read 4 KB past its end by the last QKV MMA
  s.act = o;       o += (d / 64) * kActAtom;   // fp16 x, swizzled (B operand of QKV, gate/up)
  s.qbuf = o;      o += kTokTile * kQS * 2;    // q of this head; in phase B the swizzled SwiGLU slice
  s.ownk = o;      o += kTokTile * kQS * 2;    // own keys; later the output transpose
  s.ownv = o;      o += kTokTile * kQS * 2;    // own values
  o = (o + 1023) & ~1023;
  s.tile = o;      o += 2 * kKeyTile * kD * 2; // the merged o_h, swizzled (B operand of W_o)
  s.recv = o;      o += kCl * kRecvBytes;      // split partials / gate-up partials received
  s.recv_lse = o;  o += kCl * kRowsPerRank * 4;
  s.total = o + 1024;                          // + alignment slack of the dynamic base
  return s;
}

__device__ __forceinline__ float4 ld_cg4(const float* p) { return __ldcg(reinterpret_cast<const float4*>(p)); }

__device__ __forceinline__ void red_add_v4(float* addr, float4 v) {
  asm volatile("red.relaxed.gpu.global.add.v4.f32 [%0], {%1,%2,%3,%4};" ::"l"(addr), "f"(v.x), "f"(v.y), "f"(v.z),
               "f"(v.w)
               : "memory");
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

// Arm an exchange barrier (count 1) for its next phase: the arrival plus the
// bytes the partners will deliver by st.async.
__device__ __forceinline__ void arm(uint64_t* bar, uint32_t bytes) { mbar_arrive_expect_tx(bar, bytes); }

// tensor memory -> registers: N (16 or 32) consecutive fp32 columns of each of the four
// accumulators, all loads in flight before one wait, added in accumulator order
template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t (&r)[N]);
template <>
__device__ __forceinline__ void tmem_ld_cols<16>(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
template <>
__device__ __forceinline__ void tmem_ld_cols<32>(uint32_t taddr, uint32_t (&r)[32]) {
  tmem_ld32_issue(taddr, r);
}
// the wait for every TMEM load of this thread; the registers are tied to it so that
// no use of them is scheduled before it (the first wait completes all loads)
__device__ __forceinline__ void tmem_wait_tied(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15])
               :
               : "memory");
}
__device__ __forceinline__ void tmem_wait_tied(uint32_t (&r)[32]) { tmem_wait_ld32(r); }
template <int N>
__device__ __forceinline__ void tmem_ld_sum4(uint32_t taddr, float (&v)[N]) {
  uint32_t r[kNAcc][N];
#pragma unroll
  for (int a = 0; a < kNAcc; ++a) tmem_ld_cols<N>(taddr + static_cast<uint32_t>(a) * kAccCols, r[a]);
#pragma unroll
  for (int a = 0; a < kNAcc; ++a) tmem_wait_tied(r[a]);
#pragma unroll
  for (int i = 0; i < N; ++i)
    v[i] = ((__uint_as_float(r[0][i]) + __uint_as_float(r[1][i])) + __uint_as_float(r[2][i])) + __uint_as_float(r[3][i]);
}

// Bounded wait until *counter >= target (one thread polls, the CTA follows), giving up
// after limit_ns of globaltimer (checked after every failed poll: one poll is an L2 round
// trip, far longer than the timer read). Once a wait of this CTA has timed out (*abort
// set), later waits return at once, so a broken tick still ends within about a second
// per CTA.
__device__ __forceinline__ void wait_counter(const int* counter, int target, int* status, volatile int* abort,
                                             unsigned long long limit_ns) {
  if (threadIdx.x == 0 && *abort == 0) {
    const unsigned long long t0 = global_timer_ns();
    for (;;) {
      int v;
      asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(counter) : "memory");
      if (v >= target) break;
      if (global_timer_ns() - t0 > limit_ns) {
        set_status(status, kStatusTimeout);
        *abort = 1;
        break;
      }
    }
  }
  __syncthreads();
}

template <typename CT>
__global__ void __cluster_dims__(kCl, 1, 1) __launch_bounds__(kThr, 1) persistent_tick_kernel(const PersistArgs p) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // the swizzled operand images need 1024-byte aligned shared addresses
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const Smem L = smem_layout(p.d);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bars);  // [kSlots] weight ring
  uint64_t* mma_bar = full + kSlots;   // the four issuing warps' MMA groups
  uint64_t* xbar = mma_bar + 1;        // [4] x quarter + partial sums of x^2 from rank s (phase A)
  uint64_t* qbar = xbar + kCl;         // q (and own k / v) from the partners
  uint64_t* rsbar = qbar + 1;          // split partials of the rows this CTA merges
  uint64_t* agbar = rsbar + 1;         // merged o_h rows of the partners
  uint64_t* bbar = agbar + 1;          // phase B: partial sums of x^2 and gate/up partials
  uint64_t* hbar = bbar + 1;           // phase B: the partners' SwiGLU columns
  uint64_t* drain_bar = hbar + 1;      // the four issuing threads' last MMAs (before TMEM is freed)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);  // a wait of this CTA timed out
  float* gss = reinterpret_cast<float*>(smem + L.gss);
  float* rstd = reinterpret_cast<float*>(smem + L.rstd);
  unsigned char* ring = smem + L.ring;
  unsigned char* act = smem + L.act;
  __half* qbuf = reinterpret_cast<__half*>(smem + L.qbuf);
  __half* ownk = reinterpret_cast<__half*>(smem + L.ownk);
  __half* ownv = reinterpret_cast<__half*>(smem + L.ownv);
  unsigned char* hsl = smem + L.qbuf;  // phase B: swizzled [48 tokens x 64] SwiGLU slice of the cluster
  unsigned char* obuf = smem + L.tile;  // merged o_h, swizzled [48 tokens x 128]
  float* recv = reinterpret_cast<float*>(smem + L.recv);
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
  const int d = p.d;                             // 512 (checked on the host)
  const int T = p.n_action + p.n_frame;
  const int HD = p.H * kD;
  const bool in_b = head < p.n_b_clusters;       // phase B participant (whole clusters)
  const int n_b_ctas = p.n_b_clusters * kCl;
  const int total_chunks = p.n_layers * kLayerChunks;

  // ---- ring: position q of this CTA's stream uses slot q % kSlots; per layer
  // positions 0-7 are phase-A images, 8-10 phase-B images, the rest empty
  auto chunk_src = [&](int q) -> const unsigned char* {
    const int layer = q / kLayerChunks;
    const int i = q - layer * kLayerChunks;
    const unsigned char* base = p.warena + static_cast<size_t>(layer) * p.layer_bytes;
    if (i < kPersistAChunks) return base + static_cast<size_t>(cta) * p.a_cta_bytes + static_cast<size_t>(i) * kSlotBytes;
    return base + p.b_offset + static_cast<size_t>(cta) * p.b_cta_bytes +
           static_cast<size_t>(i - kPersistAChunks) * kSlotBytes;
  };
  auto is_empty = [&](int q) {
    const int i = q % kLayerChunks;
    return i >= kPersistAChunks + (in_b ? kPersistBChunks : 0);
  };
  int issued_upto = 0;  // thread 0: ring positions issued so far (in increasing order)
  auto issue = [&](int q) {  // one thread; an empty position just completes the slot's phase
    if (q >= total_chunks || *abort) return;  // after a timeout no new copy starts
    issued_upto = q + 1;
    uint64_t* bar = full + (q % kSlots);
    if (is_empty(q)) {
      mbar_arrive(bar);
      return;
    }
    mbar_arrive_expect_tx(bar, kSlotBytes);
    bulk_g2s(ring + static_cast<size_t>(q % kSlots) * kSlotBytes, chunk_src(q), kSlotBytes, bar);
  };
  // wait for position q; false after a timeout of this tick (no MMA then reads the slot)
  auto wait_chunk = [&](int q) -> bool {
    if (*abort) return false;
    const bool ok = mbar_wait(full + (q % kSlots), static_cast<uint32_t>((q / kSlots) & 1), p.status);
    if (!ok) *abort = 1;
    return ok;
  };
  // wait for phase `parity` of an exchange barrier; false after a timeout of this tick
  auto xwait = [&](uint64_t* bar, int parity) -> bool {
    if (*abort) return false;
    const bool ok = mbar_wait_cluster(bar, static_cast<uint32_t>(parity & 1), p.status);
    if (!ok) *abort = 1;
    return ok;
  };
  uint32_t n_mma = 0;  // completed MMA groups (phase of mma_bar)
  // all threads: wait for the MMA groups just committed, then order TMEM reads after them
  auto wait_mma = [&]() {  // this CTA's own MMAs always complete: waited even after a timeout
    if (!mbar_wait(mma_bar, n_mma & 1u, p.status)) *abort = 1;
    ++n_mma;
    tc_fence_after();
  };

  // ---- exchange byte counts, identical in every layer (recomputed at each use from the
  // launch parameters rather than held in registers across the attention)
#define FSX_T (p.n_action + p.n_frame)
#define FSX_X_BYTES static_cast<uint32_t>(FSX_T * (128 * 2 + 4))  // fp16 x quarter + partial sums, per partner
#define FSX_RS_BYTES static_cast<uint32_t>((kCl - 1) * (kRecvBytes + kRowsPerRank * 4))
#define FSX_AG_BYTES static_cast<uint32_t>((kCl - 1) * kRowsPerRank * kD * 2)
#define FSX_B_BYTES static_cast<uint32_t>((kCl - 1) * (kRsBytes + FSX_T * 4))
#define FSX_H_BYTES static_cast<uint32_t>((kCl - 1) * FSX_T * 32)
#define FSX_Q_BYTES static_cast<uint32_t>((kCl - 1) * FSX_T * 64 * (rank == own_rank ? 3 : 1))

  if (tid == 0) {
    *abort = 0;
    for (int i = 0; i < kSlots; ++i) mbar_init(full + i, 1);
    mbar_init(mma_bar, kNAcc);
    for (int i = 0; i < kCl + 5; ++i) mbar_init(xbar + i, 1);
    mbar_init(drain_bar, kNAcc);
    for (int q = 0; q < kSlots; ++q) issue(q);
  }

  // ---- vehicle 0's cache range, checked once (uniform across the grid)
  const int64_t* offs = p.targs->offsets;
  const long long o_lo = p.targs->starts != nullptr ? p.targs->starts[0] : offs[0];
  const long long o_hi = o_lo + (offs[1] - offs[0]);
  bool bad = o_lo < 0 || o_hi < o_lo || o_hi > p.max_total;
  if (!bad && o_hi > o_lo)  // a non-empty cache needs every layer's rows
    for (int l = 0; l < p.n_layers; ++l)
      bad = bad || p.targs->k_cache[l] == nullptr || p.targs->v_cache[l] == nullptr;
  cluster.sync();  // barrier initialisation visible to the partners before any st.async
  if (bad) {
    if (cta == 0 && tid == 0) set_status(p.status, kStatusDeviceArg);
    if (tid == 0)
      for (int q = 0; q < kSlots && q < total_chunks; ++q) wait_chunk(q);  // let in-flight copies land
    return;
  }

  // ---- tensor memory for the four accumulators (one CTA per SM: never contended)
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  // token rows T..47 of the activation image start at zero
  for (int i = tid; i < (kTokTile - T) * (d / 8); i += kThr) {
    const int r = T + i / (d / 8);
    const int k = (i % (d / 8)) * 8;
    *reinterpret_cast<uint4*>(act + sw128_offset(kTokTile, r, k)) = make_uint4(0u, 0u, 0u, 0u);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(tmem_slot);
  const uint32_t ring_a = smem_addr(ring);
  const uint32_t act_a = smem_addr(act);
  // one MMA-issuing warp: K steps kk0 .. kk0 + nk - 1 (K = 16 each) of one 64-wide K
  // slice into accumulator `acc`: D[128 x 48] (+)= A[128 rows] . B[48 tokens]^T
  auto mma_k = [&](int acc, uint32_t a_addr, uint32_t b_addr, int kk0, int nk, bool first) {
    for (int kk = kk0; kk < kk0 + nk; ++kk)
      umma_f16(tmem + static_cast<uint32_t>(acc) * kAccCols, sw128_desc(a_addr + kk * 32),
               sw128_desc(b_addr + kk * 32), kIdesc, (first && kk == kk0) ? 0u : 1u);
  };

  const long long Lc = o_hi - o_lo;

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

  // This thread's share of a CTA's 128 columns of x when they are converted to fp16:
  // 8-column unit xu of rows xr0, xr0 + 16, xr0 + 32.
  const int xu = tid & 15;
  const int xr0 = tid >> 4;
  // this thread's fp32 columns of x (issued first thing after a phase's wait)
  auto load_x = [&](const float* Xs, int col0, float4 (&xv)[3][2]) {
#pragma unroll
    for (int i = 0; i < 3; ++i) {
      const int r = xr0 + 16 * i;
#pragma unroll
      for (int h = 0; h < 2; ++h)
        xv[i][h] = r < T ? ld_cg4(Xs + static_cast<size_t>(r) * d + col0 + xu * 8 + 4 * h) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  };
  // those columns -> fp16 x image (local, and the partners when `send_x`), per-token
  // partial sums of x^2 -> gss[rank] here and in the partners; the partners'
  // `peer_bar` counts the bytes
  auto convert_send = [&](const float4 (&xv)[3][2], int k0, bool send_x, uint64_t* peer_bar) {
#pragma unroll
    for (int i = 0; i < 3; ++i) {
      const int r = xr0 + 16 * i;
      const float4 a = xv[i][0], b = xv[i][1];
      float ss = a.x * a.x + a.y * a.y + a.z * a.z + a.w * a.w + b.x * b.x + b.y * b.y + b.z * b.z + b.w * b.w;
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);  // the row's 16 threads
      if (r < T && *abort == 0) {
        const uint4 h = make_uint4(pack_half2(a.x, a.y), pack_half2(a.z, a.w), pack_half2(b.x, b.y), pack_half2(b.z, b.w));
        unsigned char* dst = act + sw128_offset(kTokTile, r, k0 + xu * 8);
        *reinterpret_cast<uint4*>(dst) = h;
        if (xu == 0) gss[rank * kTokTile + r] = ss;
#pragma unroll
        for (int pi = 1; pi < kCl; ++pi) {
          const int peer = (rank + pi) & (kCl - 1);
          const uint32_t pb = cluster_addr(peer_bar, peer);
          if (send_x) st_async_v4(cluster_addr(dst, peer), h, pb);
          if (xu == 0) st_async_b32(cluster_addr(gss + rank * kTokTile + r, peer), __float_as_uint(ss), pb);
        }
      }
    }
  };
  // 1 / rms of every token from the four ranks' partial sums (rank order)
  auto compute_rstd = [&]() {
    if (tid < T) {
      const float ss = ((gss[tid] + gss[kTokTile + tid]) + gss[2 * kTokTile + tid]) + gss[3 * kTokTile + tid];
      rstd[tid] = rsqrtf(ss / static_cast<float>(d) + 1e-6f);
    }
  };
  // a CTA's [48 x 128] transposed output (dstT) added into X_next columns col0..col0+127,
  // plus the residual `res` when given: warp w takes rows w, w + 8, ..., lane l columns
  // 4l..4l+3, so every vector atomic of a warp covers one contiguous 512-byte row
  auto scatter_add = [&](float* Xn, int col0, const float4 (&res)[6], bool add_residual) {
#pragma unroll
    for (int i = 0; i < 6; ++i) {
      const int t = warp + 8 * i;
      if (t < T) {
        float4 v = *reinterpret_cast<const float4*>(dstT + t * kDS + lane * 4);
        if (add_residual) {
          v.x += res[i].x;
          v.y += res[i].y;
          v.z += res[i].z;
          v.w += res[i].w;
        }
        red_add_v4(Xn + static_cast<size_t>(t) * d + col0 + lane * 4, v);
      }
    }
  };
  auto load_residual = [&](const float* Xs, int col0, float4 (&res)[6]) {
#pragma unroll
    for (int i = 0; i < 6; ++i) {
      const int t = warp + 8 * i;
      res[i] = t < T ? ld_cg4(Xs + static_cast<size_t>(t) * d + col0 + lane * 4) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  };
  // the four accumulators' sum (128 output columns x 48 tokens) -> dstT[token][column];
  // warps 0-3 take tokens 0-31, warps 4-7 tokens 32-47 of their 32 TMEM lanes
  auto tmem_to_dstT = [&]() {
    const int col = (warp & 3) * 32 + lane;
    const uint32_t taddr = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
    if (warp < 4) {
      float v[32];
      tmem_ld_sum4<32>(taddr, v);
#pragma unroll
      for (int j = 0; j < 32; ++j) dstT[j * kDS + col] = v[j];
    } else {
      float v[16];
      tmem_ld_sum4<16>(taddr + 32u, v);
#pragma unroll
      for (int j = 0; j < 16; ++j) dstT[(32 + j) * kDS + col] = v[j];
    }
    tc_fence_before();
    __syncthreads();
  };

  // ---- this CTA's cache rows of a layer, staged in the shared memory that is idle
  // from the end of the QKV MMA to the end of the attention: ring slots 2-5 and
  // the activation image behind them (112 KB, contiguous). It is cut into kNB
  // buffers of kStageKeys keys (K rows then V rows, each row padded to kRowStride
  // bytes so ldmatrix reads are conflict-free), so kNB - 1 chunks are in flight
  // while one is consumed. Rows arrive raw (bf16 / fp32) by 16-byte cp.async
  // copies and are converted to fp16 in place (at the start of the row). Thread
  // t always handles 16-byte units t, t + 256, ... of a buffer (row = unit >> s,
  // no division), and the weight copies of positions 8-11 of the layer (slots
  // 2-5) are issued only once the attention is done with the region.
  constexpr int kRowStride = sizeof(CT) == 2 ? kD * 2 + 16 : kD * 4 + 16;  // 272 / 528 bytes
  constexpr int kNB = 3;                                                  // staging buffers
  constexpr int kStageRegion = 4 * kSlotBytes + 8 * kActAtom;             // 112 KB (d = 512)
  constexpr int kStageKeys = sizeof(CT) == 2 ? 64 : 36;                   // two whole key tiles (bf16)
  constexpr int kBufBytes = 2 * kStageKeys * kRowStride;                  // 34 / 37.1 KB
  constexpr int kUnitsPerRow = kD * static_cast<int>(sizeof(CT)) / 16;   // raw 16-byte units: 16 / 32
  constexpr int kUnitShift = sizeof(CT) == 2 ? 4 : 5;
  constexpr int kRawIters = (2 * kStageKeys * kUnitsPerRow + kThr - 1) / kThr;  // 8 / 9
  constexpr int kCvtIters = (2 * kStageKeys * 16 + kThr - 1) / kThr;            // fp16 units: 8 / 5
  static_assert(kSlots == 6 && kPersistAChunks == 8, "staging assumes slots 2-5 hold positions 8-11");
  static_assert((1 << kUnitShift) == kUnitsPerRow, "unit shift");
  static_assert(kBufBytes % 16 == 0 && (kStageKeys * kRowStride) % 16 == 0, "cp.async / ldmatrix alignment");
  static_assert(kNB * kBufBytes <= kStageRegion, "staging buffers exceed slots 2-5 + the activation image");
  static_assert(sizeof(CT) == 4 || kStageKeys % (2 * kKeyTile) == 0, "an even number of key tiles per bf16 chunk");
  static_assert(3 * 2 * 8 * 32 * 16 + 3 * 2 * 32 * 16 <= 8 * kActAtom, "key-half merge scratch exceeds the activation image");
  unsigned char* const stage_base = ring + 2 * kSlotBytes;  // the activation image follows the ring
  // Keys of this CTA: the cache in whole staging chunks, split near-evenly over the
  // cluster (later ranks take the extra chunks; only the last chunk can be short), and
  // all T own keys on the rank with the fewest cache keys (the last such rank), so that
  // no rank pays a chunk iteration for a few leftover keys.
  const long long n_cchunks = (Lc + kStageKeys - 1) / kStageKeys;
  auto cache_lo = [&](int r) { return min(Lc, n_cchunks * r / kCl * kStageKeys); };
  int own_rank = 0;
  for (int r = 1; r < kCl; ++r)
    if (cache_lo(r + 1) - cache_lo(r) <= cache_lo(own_rank + 1) - cache_lo(own_rank)) own_rank = r;
  const long long kbeg = cache_lo(rank);                                // first cache key of this CTA
  const int n_cache = static_cast<int>(cache_lo(rank + 1) - kbeg);      // cache keys of this CTA
  const int n_chunks = (n_cache + kStageKeys - 1) / kStageKeys;
  const int own_lo = 0;                                                 // own keys of this CTA
  const int own_n = rank == own_rank ? T : 0;
  const size_t tok_bytes = static_cast<size_t>(p.H) * kD * sizeof(CT);  // one token row of all heads
  const size_t head_off = (static_cast<size_t>(o_lo + kbeg) * p.H + head) * kD * sizeof(CT);
  // all threads: 16-byte cp.async copies of chunk j into buffer j % kNB (one commit group)
  auto stage_issue = [&](int j, const unsigned char* kh, const unsigned char* vh) {
    const int k0 = j * kStageKeys;
    const int n = min(kStageKeys, n_cache - k0);
    unsigned char* kb = stage_base + (j % kNB) * kBufBytes;
#pragma unroll
    for (int it = 0; it < kRawIters; ++it) {
      const int i = tid + it * kThr;
      const int r = i >> kUnitShift;  // row of [K rows ; V rows]
      const int u = i & (kUnitsPerRow - 1);
      const bool is_v = r >= kStageKeys;
      const int key = is_v ? r - kStageKeys : r;
      if (r < 2 * kStageKeys && key < n)
        cp_async_16(smem_addr(kb + r * kRowStride + u * 16),
                    (is_v ? vh : kh) + static_cast<size_t>(k0 + key) * tok_bytes + u * 16);
    }
    cp_async_commit();
  };
  uint32_t range_seen = 0;  // a cache value outside the fp16 range was saturated
  // all threads: wait for chunk j and convert it to fp16 in place
  auto stage_ready = [&](int j) {
    const int younger = min(n_chunks - 1 - j, kNB - 1);  // groups of later chunks still in flight
    if (younger >= 2)
      cp_async_wait<2>();
    else if (younger == 1)
      cp_async_wait<1>();
    else
      cp_async_wait<0>();
    // bf16: a thread converts exactly the units it copied (same unit -> thread map), so
    // its own wait suffices; fp32 units are regrouped and need every thread's copies
    if (sizeof(CT) != 2) __syncthreads();
    const int n = min(kStageKeys, n_cache - j * kStageKeys);
    unsigned char* kb = stage_base + (j % kNB) * kBufBytes;
    if (sizeof(CT) == 2) {
      // two rounds of half the units, every load of a round before its first store
      constexpr int kHalf = (kCvtIters + 1) / 2;
#pragma unroll
      for (int r0 = 0; r0 < kCvtIters; r0 += kHalf) {
        uint4 v[kHalf];
#pragma unroll
        for (int it = 0; it < kHalf; ++it) {
          const int i = tid + (r0 + it) * kThr;
          const int r = i >> 4;
          const int key = r >= kStageKeys ? r - kStageKeys : r;
          if (r0 + it < kCvtIters && r < 2 * kStageKeys && key < n)
            v[it] = *reinterpret_cast<const uint4*>(kb + r * kRowStride + (i & 15) * 16);
        }
#pragma unroll
        for (int it = 0; it < kHalf; ++it) {
          const int i = tid + (r0 + it) * kThr;
          const int r = i >> 4;
          const int key = r >= kStageKeys ? r - kStageKeys : r;
          if (r0 + it < kCvtIters && r < 2 * kStageKeys && key < n)
            *reinterpret_cast<uint4*>(kb + r * kRowStride + (i & 15) * 16) =
                make_uint4(bf16x2_to_half2_sat(v[it].x, range_seen), bf16x2_to_half2_sat(v[it].y, range_seen),
                           bf16x2_to_half2_sat(v[it].z, range_seen), bf16x2_to_half2_sat(v[it].w, range_seen));
        }
      }
    } else {
      // 32-byte fp32 unit u of a row -> 16-byte fp16 unit u at the row start. A row's 16
      // units fall in one round of 256, all reads of a round land before its writes, and
      // a unit's input is never written by a later round.
#pragma unroll 1
      for (int it = 0; it < kCvtIters; ++it) {
        const int i = tid + it * kThr;
        const int r = i >> 4;
        const int key = r >= kStageKeys ? r - kStageKeys : r;
        const bool live = r < 2 * kStageKeys && key < n;
        unsigned char* row = kb + r * kRowStride;
        const int u = i & 15;
        uint4 o = make_uint4(0u, 0u, 0u, 0u);
        if (live) {
          const float4 a = *reinterpret_cast<const float4*>(row + u * 32);
          const float4 b = *reinterpret_cast<const float4*>(row + u * 32 + 16);
          o = make_uint4(f32x2_to_half2_sat(a.x, a.y, range_seen), f32x2_to_half2_sat(a.z, a.w, range_seen),
                         f32x2_to_half2_sat(b.x, b.y, range_seen), f32x2_to_half2_sat(b.z, b.w, range_seen));
        }
        __syncthreads();
        if (live) *reinterpret_cast<uint4*>(row + u * 16) = o;
        __syncthreads();
      }
    }
    __syncthreads();
  };

  // ---- arm the exchange barriers for layer 0, then publish the token assembly
  if (tid < kTokTile) rstd[tid] = 0.f;  // padding tokens T..47 stay at zero
  if (tid == 0) {
    for (int s_ = 1; s_ < kCl; ++s_) arm(xbar + ((rank + s_) & (kCl - 1)), FSX_X_BYTES);
    arm(qbar, FSX_Q_BYTES);
    arm(rsbar, FSX_RS_BYTES);
    arm(agbar, FSX_AG_BYTES);
    if (in_b) {
      arm(bbar, FSX_B_BYTES);
      arm(hbar, FSX_H_BYTES);
    }
  }
  arrive(p.counters + 0);

  // this CTA's share of the residual buffer each phase zeroes
  const int zA0 = static_cast<int>(static_cast<long long>(n_elem) * cta / G);
  const int zA1 = static_cast<int>(static_cast<long long>(n_elem) * (cta + 1) / G);
  const int zB0 = static_cast<int>(static_cast<long long>(n_elem) * cta / n_b_ctas);
  const int zB1 = static_cast<int>(static_cast<long long>(n_elem) * (cta + 1) / n_b_ctas);

  int q0 = 0;  // first ring position of the current layer
  const float scale_log2 = 1.4426950408889634f * rsqrtf(static_cast<float>(kD));

  for (int layer = 0; layer < p.n_layers; ++layer, q0 += kLayerChunks) {
    const int par = layer & 1;  // phase of every exchange barrier in this layer
    const int sA = 2 * layer;
    float* Xc = X0 + static_cast<size_t>(sA % 3) * xs;        // layer input
    float* Xm = X0 + static_cast<size_t>((sA + 1) % 3) * xs;  // after attention
    float* Xz = X0 + static_cast<size_t>((sA + 2) % 3) * xs;  // zeroed now, written by phase B
    // this CTA's first cache row (head h, key kbeg of the vehicle) in layer l's K and V
    const unsigned char* kc = n_chunks > 0 ? static_cast<const unsigned char*>(p.targs->k_cache[layer]) + head_off : nullptr;
    const unsigned char* vc = n_chunks > 0 ? static_cast<const unsigned char*>(p.targs->v_cache[layer]) + head_off : nullptr;

    // =========================== phase A ===========================
    wait_counter(p.counters + sA, sA == 0 ? G : n_b_ctas, p.status, abort, p.wait_limit_ns);
    {
      float4 xv[3][2];
      load_x(Xc, rank * 128, xv);
      // zero the buffer phase B accumulates into (while the loads are in flight)
      for (int e = zA0 + tid; e < zA1; e += kThr) __stcg(Xz + e, 0.f);
      // this rank's 128 columns of x -> fp16 image here and in the partners (K slices
      // 2 rank, 2 rank + 1), partial sums of x^2 to every rank
      convert_send(xv, rank * 128, true, xbar + rank);
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // the local quarter -> tensor core
    __syncthreads();

    // --- QKV: D[96 (+32 unused) rows x 48 tokens] over K = 512. Warp w < 4 runs K quarter w
    // (slices 2w, 2w + 1: rank w's columns of x) into accumulator w as soon as rank w's
    // columns and the weight slots under them have arrived; the 12 KB K slices lie back
    // to back in slots 0-5
    if (warp < kNAcc) {
      tc_fence_after();
      const int a0 = 2 * warp;
      bool ok = true;
      for (int sl = (a0 * kQkvAtom) / kSlotBytes; sl <= ((a0 + 2) * kQkvAtom - 1) / kSlotBytes; ++sl)
        ok = wait_chunk(q0 + sl) && ok;
      if (warp != rank) ok = xwait(xbar + warp, par) && ok;
      if (ok && lane == 0) {
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // the partner's columns -> tensor core
        mma_k(warp, ring_a + a0 * kQkvAtom, act_a + a0 * kActAtom, 0, 4, true);
        mma_k(warp, ring_a + (a0 + 1) * kQkvAtom, act_a + (a0 + 1) * kActAtom, 0, 4, false);
      }
      __syncwarp();
      if (lane == 0) umma_commit(mma_bar);
      __syncwarp();
    }
    // every partner's partial sums of x^2 have arrived: 1 / rms per token; re-arm for the next layer
    for (int s_ = 1; s_ < kCl; ++s_) xwait(xbar + ((rank + s_) & (kCl - 1)), par);
    if (tid == 0 && *abort == 0)
      for (int s_ = 1; s_ < kCl; ++s_) arm(xbar + ((rank + s_) & (kCl - 1)), FSX_X_BYTES);
    compute_rstd();
    __syncthreads();
    wait_mma();
    for (int j = 0; j < kNB && j < n_chunks; ++j)  // slots 2-5 and the activation image are free
      stage_issue(j, kc, vc);
    // rows 32j..32j+31 of the accumulators are q, k, v dims 32 rank .. 32 rank + 31,
    // scaled by 1 / rms of their token
    if ((warp & 3) < 3) {
      const int kind = warp & 3;
      __half* b = kind == 0 ? qbuf : (kind == 1 ? ownk : ownv);
      const int dim = rank * 32 + lane;
      const uint32_t taddr = tmem + (static_cast<uint32_t>(kind * 32) << 16);
      const int c_lo = warp < 4 ? 0 : 32;
      const int c_hi = warp < 4 ? 32 : 48;
      if (warp < 4) {
        float v[32];
        tmem_ld_sum4<32>(taddr, v);
#pragma unroll
        for (int j = 0; j < 32; ++j) b[j * kQS + dim] = __float2half_rn(v[j] * rstd[j]);
      } else {
        float v[16];
        tmem_ld_sum4<16>(taddr + 32u, v);
#pragma unroll
        for (int j = 0; j < 16; ++j) b[(32 + j) * kQS + dim] = __float2half_rn(v[j] * rstd[32 + j]);
      }
      __syncwarp();
      // this warp's token rows below T (dims 32 rank .. + 31, four 16-byte units a row): q to
      // every partner, own k and v to the rank that attends over the own keys
      if (*abort == 0 && (kind == 0 || own_rank != rank)) {
        for (int i = lane; i < (min(c_hi, T) - c_lo) * 4; i += 32) {
          const __half* src = b + (c_lo + (i >> 2)) * kQS + rank * 32 + (i & 3) * 8;
          const uint4 v = *reinterpret_cast<const uint4*>(src);
          if (kind == 0) {
#pragma unroll
            for (int pi = 1; pi < kCl; ++pi) {
              const int peer = (rank + pi) & (kCl - 1);
              st_async_v4(cluster_addr(src, peer), v, cluster_addr(qbar, peer));
            }
          } else {
            st_async_v4(cluster_addr(src, own_rank), v, cluster_addr(qbar, own_rank));
          }
        }
      }
    }
    tc_fence_before();
    __syncthreads();
    if (tid == 0)  // slots 0, 1 are free: W_o of this layer (slots 2-5 stage the cache)
      for (int i = kSlots; i < kPersistAChunks; ++i) issue(q0 + i);
    xwait(qbar, par);  // q (and on the own-key rank, own k / v) of every partner
    if (tid == 0 && *abort == 0) arm(qbar, FSX_Q_BYTES);

    // --- Eq. 1 over this CTA's cache keys, then its own keys, in 32-key tiles. Warp w < 6
    // takes query rows 16 (w % 3) .. +15 and every other key tile (tiles kh, kh + 2, ...
    // of a chunk, kh = w / 3) over all 128 value dims; the two key halves of a query
    // tile are merged in shared memory afterwards (log-sum-exp weights).
    const int qt = warp % 3;
    const int kh = warp / 3;
    float o_acc[16][4];
    float m_run[2] = {-CUDART_INF_F, -CUDART_INF_F};
    float l_run[2] = {0.f, 0.f};
#pragma unroll
    for (int nb = 0; nb < 16; ++nb)
#pragma unroll
      for (int e = 0; e < 4; ++e) o_acc[nb][e] = 0.f;
    uint32_t qf[8][4];
    if (warp < 6) {
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const __half* src = qbuf + static_cast<size_t>(qt * 16 + (lane & 15)) * kQS + kk * 16 + (lane >> 4) * 8;
        ldsm_x4(qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3], smem_addr(src));
      }
    }
    // this warp's key tiles of keys 0..n-1, K rows at kb and V rows at vb (fp16, `stride` bytes apart)
    auto attend = [&](const unsigned char* kb, const unsigned char* vb, int stride, int n) {
      for (int t0 = kh * kKeyTile; t0 < n; t0 += 2 * kKeyTile) {
        const int rows = min(kKeyTile, n - t0);
        float sc[4][4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
#pragma unroll
          for (int e = 0; e < 4; ++e) sc[j][e] = 0.f;
          int r = t0 + j * 8 + (lane & 7);
          r = r < n ? r : 0;  // masked below; any valid row keeps the products finite
          const uint32_t krow = smem_addr(kb + r * stride);
#pragma unroll
          for (int dd = 0; dd < 4; ++dd) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4(b0, b1, b2, b3, krow + (dd * 4 + (lane >> 3)) * 16);
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
        for (int nb = 0; nb < 16; ++nb) {
          o_acc[nb][0] *= alpha[0];
          o_acc[nb][1] *= alpha[0];
          o_acc[nb][2] *= alpha[1];
          o_acc[nb][3] *= alpha[1];
        }
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
          int r = t0 + kk * 16 + (lane & 7) + 8 * ((lane >> 3) & 1);
          r = r < n ? r : 0;
          const uint32_t vrow = smem_addr(vb + r * stride);
#pragma unroll
          for (int np = 0; np < 8; ++np) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4_trans(b0, b1, b2, b3, vrow + (np * 2 + (lane >> 4)) * 16);
            mma_f16_16816(o_acc[2 * np], pf[kk][0], pf[kk][1], pf[kk][2], pf[kk][3], b0, b1);
            mma_f16_16816(o_acc[2 * np + 1], pf[kk][0], pf[kk][1], pf[kk][2], pf[kk][3], b2, b3);
          }
        }
      }
    };
    for (int j = 0; j < n_chunks; ++j) {
      stage_ready(j);
      if (warp < 6) {
        const unsigned char* kb = stage_base + (j % kNB) * kBufBytes;
        attend(kb, kb + kStageKeys * kRowStride, kRowStride, min(kStageKeys, n_cache - j * kStageKeys));
      }
      __syncthreads();  // buffer j % kNB consumed
      if (j + kNB < n_chunks) stage_issue(j + kNB, kc, vc);
    }
    if (tid == 0) {  // every staged row has landed and been read: gate/up, W_d into slots 2-5
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      for (int i = kPersistAChunks; i < kLayerChunks; ++i) issue(q0 + i);
    }
    if (warp < 6 && own_n > 0)
      attend(reinterpret_cast<const unsigned char*>(ownk + static_cast<size_t>(own_lo) * kQS),
             reinterpret_cast<const unsigned char*>(ownv + static_cast<size_t>(own_lo) * kQS), kQS * 2, own_n);

    // --- merge the two key halves of each query tile: warp (qt, kh) keeps value dims
    // 64 kh .. 64 kh + 63. It hands the other 64 dims of its accumulator and its running
    // max / sum to its partner through the activation image (idle now; thread-fragment
    // order, so every lane reads back exactly its partner lane's values).
    float o_fin[8][4];
    {
      float4* xo = reinterpret_cast<float4*>(act);   // [3 qt][2 kh][8][32 lanes]
      float4* xml = xo + 3 * 2 * 8 * 32;              // [3 qt][2 kh][32 lanes]: m0, m1, l0, l1
      if (warp < 6) {
#pragma unroll
        for (int nb = 0; nb < 8; ++nb) {
          const float* src = kh == 0 ? o_acc[8 + nb] : o_acc[nb];
          xo[((qt * 2 + kh) * 8 + nb) * 32 + lane] = make_float4(src[0], src[1], src[2], src[3]);
        }
        xml[(qt * 2 + kh) * 32 + lane] = make_float4(m_run[0], m_run[1], l_run[0], l_run[1]);
      }
      __syncthreads();
      if (warp < 6) {
        const int pk = 1 - kh;
        const float4 pml = xml[(qt * 2 + pk) * 32 + lane];
        const float pm[2] = {pml.x, pml.y};
        const float pl[2] = {pml.z, pml.w};
        float sa[2], sb[2];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const float m = fmaxf(m_run[r], pm[r]);
          sa[r] = m == -CUDART_INF_F ? 0.f : exp2f(m_run[r] - m);
          sb[r] = m == -CUDART_INF_F ? 0.f : exp2f(pm[r] - m);
          l_run[r] = l_run[r] * sa[r] + pl[r] * sb[r];
          m_run[r] = m;
        }
#pragma unroll
        for (int nb = 0; nb < 8; ++nb) {
          const float4 po = xo[((qt * 2 + pk) * 8 + nb) * 32 + lane];
          const float* mine = kh == 0 ? o_acc[nb] : o_acc[8 + nb];
          o_fin[nb][0] = mine[0] * sa[0] + po.x * sb[0];
          o_fin[nb][1] = mine[1] * sa[0] + po.y * sb[0];
          o_fin[nb][2] = mine[2] * sa[1] + po.z * sb[1];
          o_fin[nb][3] = mine[3] * sa[1] + po.w * sb[1];
        }
      }
    }

    // --- merge the 4 splits: every row's normalised fp32 partial and log-sum-exp go
    // straight from the registers to the rank that owns the row (st.async to the partners)
    if (warp < 6 && *abort == 0) {
      auto put4 = [&](float* ptr, int dst, float a, float b, float c, float e) {
        if (dst == rank)
          *reinterpret_cast<float4*>(ptr) = make_float4(a, b, c, e);
        else
          st_async_v4(cluster_addr(ptr, dst),
                      make_uint4(__float_as_uint(a), __float_as_uint(b), __float_as_uint(c), __float_as_uint(e)),
                      cluster_addr(rsbar, dst));
      };
      auto put1 = [&](float* ptr, int dst, float a) {
        if (dst == rank)
          *ptr = a;
        else
          st_async_b32(cluster_addr(ptr, dst), __float_as_uint(a), cluster_addr(rsbar, dst));
      };
      const int qr0 = qt * 16 + (lane >> 2);
      const int qr1 = qr0 + 8;
      const int own0 = qr0 / kRowsPerRank;
      const int own1 = qr1 / kRowsPerRank;
      const float inv0 = l_run[0] > 0.f ? 1.f / l_run[0] : 0.f;
      const float inv1 = l_run[1] > 0.f ? 1.f / l_run[1] : 0.f;
      float* d0 = recv + (rank * kRowsPerRank + qr0 - own0 * kRowsPerRank) * kD;
      float* d1 = recv + (rank * kRowsPerRank + qr1 - own1 * kRowsPerRank) * kD;
      // lanes 2j and 2j + 1 hold columns 4j'..4j'+3 of rows qr0 and qr1 in pairs: the even
      // lane sends row qr0's four, the odd lane row qr1's (one 16-byte store each)
      const bool odd = (lane & 1) != 0;
#pragma unroll
      for (int nb = 0; nb < 8; ++nb) {
        const int c = kh * 64 + nb * 8 + 2 * (lane & 3);
        const float a0 = o_fin[nb][0] * inv0, a1 = o_fin[nb][1] * inv0;
        const float b0 = o_fin[nb][2] * inv1, b1 = o_fin[nb][3] * inv1;
        const float g0 = __shfl_xor_sync(0xffffffffu, odd ? a0 : b0, 1);
        const float g1 = __shfl_xor_sync(0xffffffffu, odd ? a1 : b1, 1);
        if (!odd)
          put4(d0 + c, own0, a0, a1, g0, g1);
        else
          put4(d1 + c - 2, own1, g0, g1, b0, b1);
      }
      if (kh == 0 && (lane & 3) == 0) {
        put1(recv_lse + rank * kRowsPerRank + qr0 - own0 * kRowsPerRank, own0,
             l_run[0] > 0.f ? m_run[0] + log2f(l_run[0]) : -CUDART_INF_F);
        put1(recv_lse + rank * kRowsPerRank + qr1 - own1 * kRowsPerRank, own1,
             l_run[1] > 0.f ? m_run[1] + log2f(l_run[1]) : -CUDART_INF_F);
      }
    }
    xwait(rsbar, par);  // every partner's partials of the rows this CTA merges
    __syncthreads();    // and this CTA's own
    if (tid == 0 && *abort == 0) arm(rsbar, FSX_RS_BYTES);
    // merged rows of o_h -> swizzled image (the W_o B operand) here and in every partner
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
            const float4 f = *reinterpret_cast<const float4*>(recv + (s * kRowsPerRank + rr) * kD + c);
            a0 += w * f.x;
            a1 += w * f.y;
            a2 += w * f.z;
            a3 += w * f.w;
            wsum += w;
          }
        }
        const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
        uint2 out;
        out.x = pack_half2(a0 * inv, a1 * inv);
        out.y = pack_half2(a2 * inv, a3 * inv);
        unsigned char* dst = obuf + sw128_offset(kTokTile, row, c);
        *reinterpret_cast<uint2*>(dst) = out;
        if (*abort == 0) {
#pragma unroll
          for (int pi = 1; pi < kCl; ++pi) {
            const int peer = (rank + pi) & (kCl - 1);
            st_async_v2(cluster_addr(dst, peer), out.x, out.y, cluster_addr(agbar, peer));
          }
        }
        if (p.attn_capture != nullptr && row < T)
          *reinterpret_cast<uint2*>(p.attn_capture + (static_cast<size_t>(layer) * T + row) * HD + head * kD + c) = out;
      }
    }
    xwait(agbar, par);  // the partners' merged rows
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // o_h -> tensor core
    __syncthreads();
    if (tid == 0 && *abort == 0) arm(agbar, FSX_AG_BYTES);

    // --- W_o: this CTA's 128 output columns for head h, K = 128 (slots 0, 1); warp w:
    // slice w / 2, K steps 2 (w % 2) .. + 1
    if (warp < kNAcc) {
      tc_fence_after();
      const int a = warp >> 1;
      const bool ok = wait_chunk(q0 + kSlots + a);
      if (ok && lane == 0) mma_k(warp, ring_a + a * kSlotBytes, smem_addr(obuf) + a * kActAtom, (warp & 1) * 2, 2, true);
      __syncwarp();
      if (lane == 0) umma_commit(mma_bar);
      __syncwarp();
    }
    float4 res[6];
    if (head == 0) load_residual(Xc, rank * 128, res);  // cluster 0 adds the residual itself
    wait_mma();
    tmem_to_dstT();
    if (tid == 0) {  // slots 0, 1 free (all of 0-5 for CTAs without phase B): next layer's QKV
      const int n = in_b ? 2 : kSlots;
      for (int i = 0; i < n; ++i) issue(q0 + kLayerChunks + i);
    }
    scatter_add(Xm, rank * 128, res, head == 0);
    flag_range(p.status, range_seen);  // every thread's own units; published by the arrival
    arrive(p.counters + sA + 1);

    // =========================== phase B ===========================
    if (in_b) {
      const int c = head;  // SwiGLU column block 64c..64c+63
      wait_counter(p.counters + sA + 1, G, p.status, abort, p.wait_limit_ns);
      {
        float4 xv[3][2];
        load_x(Xm, rank * 128, xv);
        // zero the buffer the next phase A accumulates into (this layer's input is consumed)
        for (int e = zB0 + tid; e < zB1; e += kThr) __stcg(Xc + e, 0.f);
        // this rank's 128 columns of x -> fp16 K slices 0, 1 here (no exchange: each CTA runs
        // the gate/up MMAs over its own K quarter), partial sums of x^2 to every rank
        convert_send(xv, 0, false, bbar);
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // visible to the tensor core
      __syncthreads();
      // gate/up over this rank's K quarter: D[128 rows x 48 tokens], rows 32s..32s+31 = the
      // 16 gate and 16 up rows of rank s's SwiGLU columns (K slices in slots 2, 3); warp w:
      // slice w / 2, K steps 2 (w % 2) .. + 1
      if (warp < kNAcc) {
        tc_fence_after();
        const int a = warp >> 1;
        const bool ok = wait_chunk(q0 + kPersistAChunks + a);
        if (ok && lane == 0) mma_k(warp, ring_a + (2 + a) * kSlotBytes, act_a + a * kActAtom, (warp & 1) * 2, 2, true);
        __syncwarp();
        if (lane == 0) umma_commit(mma_bar);
        __syncwarp();
      }
      wait_mma();
      // reduce-scatter of the K partials: rows 32q..32q+31 (the accumulators' sum) go to rank q
      // as recv[this rank][row][48 tokens] (fp32)
      {
        const int q = warp & 3;
        const uint32_t taddr = tmem + (static_cast<uint32_t>(q * 32) << 16);
        float* dst = recv + (rank * 32 + lane) * kTokTile;
        auto put = [&](const float* v, int c0, int n) {
          for (int j = 0; j < n; j += 4) {
            const uint4 u = make_uint4(__float_as_uint(v[j]), __float_as_uint(v[j + 1]), __float_as_uint(v[j + 2]),
                                       __float_as_uint(v[j + 3]));
            if (q == rank)
              *reinterpret_cast<uint4*>(dst + c0 + j) = u;
            else if (*abort == 0)
              st_async_v4(cluster_addr(dst + c0 + j, q), u, cluster_addr(bbar, q));
          }
        };
        if (warp < 4) {
          float v[32];
          tmem_ld_sum4<32>(taddr, v);
          put(v, 0, 32);
        } else {
          float v[16];
          tmem_ld_sum4<16>(taddr + 32u, v);
          put(v, 32, 16);
        }
      }
      tc_fence_before();
      __syncthreads();
      if (tid == 0)  // slots 2, 3 free: next layer's QKV
        for (int i = 2; i < 4; ++i) issue(q0 + kLayerChunks + i);
      xwait(bbar, par);  // every partner's partial sums of x^2 and gate/up partials
      if (tid == 0 && *abort == 0) arm(bbar, FSX_B_BYTES);
      compute_rstd();
      __syncthreads();
      // h = silu(gate) * up for this rank's 16 SwiGLU columns: K partials summed in rank
      // order and scaled by 1 / rms; 8 columns a thread -> the swizzled slice here and in
      // every partner
      for (int i = tid; i < kTokTile * 2; i += kThr) {
        const int t = i >> 1;
        const int c8 = (i & 1) * 8;
        const float r = rstd[t];
        uint32_t hp[4];
#pragma unroll
        for (int j = 0; j < 8; j += 2) {
          float hv[2];
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int cc = c8 + j + e;
            float g = 0.f, u = 0.f;
#pragma unroll
            for (int src = 0; src < kCl; ++src) {
              g += recv[(src * 32 + cc) * kTokTile + t];
              u += recv[(src * 32 + 16 + cc) * kTokTile + t];
            }
            g *= r;
            u *= r;
            hv[e] = __fdividef(g, 1.f + __expf(-g)) * u;
          }
          hp[j >> 1] = pack_half2(hv[0], hv[1]);
        }
        const uint4 hv4 = make_uint4(hp[0], hp[1], hp[2], hp[3]);
        unsigned char* dst = hsl + sw128_offset(kTokTile, t, rank * 16 + c8);
        *reinterpret_cast<uint4*>(dst) = hv4;
        if (t < T && *abort == 0) {
#pragma unroll
          for (int pi = 1; pi < kCl; ++pi) {
            const int peer = (rank + pi) & (kCl - 1);
            st_async_v4(cluster_addr(dst, peer), hv4, cluster_addr(hbar, peer));
          }
        }
      }
      xwait(hbar, par);  // the partners' SwiGLU columns
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // the SwiGLU slice -> tensor core
      __syncthreads();
      if (tid == 0 && *abort == 0) arm(hbar, FSX_H_BYTES);
      // --- W_d: 128 output columns over the cluster's 64 SwiGLU inputs (slot 4); warp w: K step w
      if (warp < kNAcc) {
        tc_fence_after();
        const bool ok = wait_chunk(q0 + kPersistAChunks + 2);
        if (ok && lane == 0) mma_k(warp, ring_a + 4 * kSlotBytes, smem_addr(hsl), warp, 1, true);
        __syncwarp();
        if (lane == 0) umma_commit(mma_bar);
        __syncwarp();
      }
      float4 resb[6];
      if (c == 0) load_residual(Xm, rank * 128, resb);  // cluster 0 adds the residual itself
      wait_mma();
      tmem_to_dstT();
      if (tid == 0)  // slots 4, 5 free: next layer's QKV
        for (int i = 4; i < kSlots; ++i) issue(q0 + kLayerChunks + i);
      float* Xn = X0 + static_cast<size_t>((sA + 2) % 3) * xs;
      scatter_add(Xn, rank * 128, resb, c == 0);
      arrive(p.counters + sA + 2);
    }
  }

  // ---- leave nothing in flight. Every path reaches this point, a timed-out tick included
  // (its waits on other CTAs return at once). In order: this thread's cache-row copies;
  // the ring copies issued (a timed-out tick stops issuing, and may have skipped the waits
  // of the last ones: wait, bounded, for the last position of every slot); the MMAs of the
  // four issuing threads (a last commit each on drain_bar); the partners' stores into this
  // CTA's shared memory (the cluster barrier below); then the tensor memory is freed.
  cp_async_wait<0>();
  if (tid == 0)
    for (int q = issued_upto - kSlots; q < issued_upto; ++q)
      if (q >= 0 && !is_empty(q)) {
        const unsigned long long t0 = global_timer_ns();
        uint32_t done = 0;
        while (!done && global_timer_ns() - t0 < 100000000ull)
          asm volatile(
              "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
              : "=r"(done)
              : "r"(smem_addr(full + q % kSlots)), "r"(static_cast<uint32_t>((q / kSlots) & 1))
              : "memory");
      }
  if (warp < kNAcc) {
    if (lane == 0) umma_commit(drain_bar);
    __syncwarp();
  }
  mbar_wait(drain_bar, 0u, p.status);
  tc_fence_after();
  // no CTA leaves while a partner may still write into its shared memory
  cluster.sync();
  tc_fence_before();
  __syncthreads();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");

  // =========================== head ===========================
  if (cta == 0 && p.head) {
    wait_counter(p.counters + 2 * p.n_layers, n_b_ctas, p.status, abort, p.wait_limit_ns);
    // a tick with a device-side error (an out-of-range cache value, a timeout) writes no waypoint
    if (*reinterpret_cast<volatile int*>(p.status) != 0) return;
    const float* Xf = X0 + static_cast<size_t>((2 * p.n_layers) % 3) * xs;
    for (int j = warp; j < p.n_waypoints; j += kThr / 32) {
      const float* xr = Xf + static_cast<size_t>(j) * d;
      float ss = 0.f;
      for (int c = lane; c < d; c += 32) {
        const float v = __ldcg(xr + c);
        ss += v * v;
      }
      ss = warp_sum(ss);
      const float rstd_j = rsqrtf(ss / static_cast<float>(d) + 1e-6f);
      float o0 = 0.f, o1 = 0.f;
      for (int c = lane; c < d; c += 32) {
        const float n = __ldcg(xr + c) * rstd_j * p.final_norm[c];
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
#undef FSX_T
#undef FSX_X_BYTES
#undef FSX_RS_BYTES
#undef FSX_AG_BYTES
#undef FSX_B_BYTES
#undef FSX_H_BYTES
#undef FSX_Q_BYTES

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
