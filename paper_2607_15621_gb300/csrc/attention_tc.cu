// Eq. 1 of Sec. 3.1 on the 5th-generation tensor cores: one CTA per (vehicle,
// head) computes softmax(Q [K_vlm ; K_ae]^T / sqrt(128)) [V_vlm ; V_ae] for the
// expert's queries (at most 48, padded to an M = 64 tile) with a bf16 backbone
// cache, one split, fp32 accumulation. S = Q K^T in fp16: the bf16 cache K rows are
// converted in shared memory (exact for |x| in [2^-14, 65504]) by the warps that
// stage them. P V keeps the cache V rows in bf16 and splits P into bf16 P_hi + P_lo
// (16 significant bits, more than fp16's 11); the own chunk (fp16 V) splits P into
// fp16 P_hi + P_lo instead.
//
// Data path ("slot" = 64 keys; shared-memory operands 128-byte swizzled):
//   Q             [64 q][128 d] fp16   smem, A of S          (K-major)
//   K slot (x3)   [64 keys][128 d]     smem, B of S          (K-major)
//   V slot (x3)   [64 keys][128 d]     smem, B of P V        (N = d contiguous, MN-major;
//                                      bf16 cache rows, fp16 own rows)
//   S (x2)        [64 q][64 keys] fp32 tensor memory, 64 columns each
//   P_hi, P_lo    [64 q][64 keys]      tensor memory, A of P V, written over the
//                                      S buffer they were computed from (32 columns each)
//   O             [64 q][128 d] fp32   tensor memory, 128 columns
//   Row q of an M = 64 tile lives in lane (q mod 16) + 32 (q / 16).
// Chunk 0 holds the expert's own keys (fp16 as produced), chunk 1 + j the cache keys
// [64 j, 64 j + 64); chunk i sits in K / V slot i mod 3.
//
// Warp roles (256 threads): warps 0-2 run the online softmax for query rows
// 16 w .. 16 w + 15, two rows per thread; warp 3 lane 0 issues S and P V as their inputs become
// ready; warps 4-5 stage (and convert) the K rows, warps 6-7 the V rows, two chunks ahead.
// Every wait is bounded; a timeout raises the status word and the CTA drains its
// MMAs before it frees the tensor memory.
#include <cuda.h>
#include <math_constants.h>

#include "device_util.cuh"
#include "kernels.h"
#include "tcgen05.cuh"

namespace fsx {

namespace {

constexpr int kD = kHeadDim;           // 128
constexpr int kSlotKeys = 64;          // keys per chunk
constexpr int kThreadsTc = 256;
constexpr int kSoftmaxWarps = 3;       // rows 0..47
constexpr int kMmaWarp = 3;
constexpr int kProdWarp0 = 4;     // warps 4-5 stage K, warps 6-7 stage V
constexpr int kProdThreads = 64;  // per tensor
constexpr int kTmemCols = 256;         // S[2] x 64 + O 128
constexpr uint32_t kColS = 0;    // S / P buffers at columns 0 and 64
constexpr uint32_t kColO = 128;

// shared-memory layout (bytes from the 1024-aligned base)
constexpr int kQBytes = 64 * kD * 2;            // 16 KB
constexpr int kSlotBytes = kSlotKeys * kD * 2;  // 16 KB
constexpr int kSlots = 3;                       // per tensor
constexpr int kOffQ = 0;
constexpr int kOffK = kOffQ + kQBytes;
constexpr int kOffV = kOffK + kSlots * kSlotBytes;
constexpr int kOffBar = kOffV + kSlots * kSlotBytes;
// barriers: kfull[3], kempty[3], vfull[3], vempty[3], sfull[2], pfull[2], pvdone[2], drain, ktma[3], vtma[3]
constexpr int kNumBars = 25;
constexpr int kSmemTc = kOffBar + kNumBars * 8 + 8 /*tmem slot + abort*/;
static_assert(kSmemTc + 1024 <= (228 * 1024) / 2, "two CTAs per SM");

// byte offset of 16-byte unit u (8 elements) of row r in a [rows][128] tile made of
// 64-element swizzled column blocks (1024-byte atoms of 8 rows; blocks 8 KB apart
// for 64-row tiles)
__device__ __forceinline__ uint32_t tile128_off(int r, int u) {
  return (u >> 3) * 8192 + (r >> 3) * 1024 + (r & 7) * 128 + ((((u & 7) ^ (r & 7))) << 4);
}

// MN-major 128-byte-swizzled descriptor: LBO = distance between 64-element blocks
// along N, SBO = distance between 8-row groups along K
__device__ __forceinline__ uint64_t sw128_desc_mn(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

// kind::f16 instruction descriptor, fp16 A and B, fp32 D; b_mn: B is N-contiguous
__host__ __device__ constexpr uint32_t idesc_f16_mn(int m, int n, bool b_mn) {
  return (1u << 4) | (b_mn ? (1u << 16) : 0u) | (static_cast<uint32_t>(n >> 3) << 17) |
         (static_cast<uint32_t>(m >> 4) << 24);
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// two fp32 -> bf16x2 (round to nearest even), lo in the low half
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// D[tmem] (+)= A[tmem] * B[smem]^T, one K = 16 step (A: M rows in the D lane layout,
// two 16-bit values per column)
__device__ __forceinline__ void umma_f16_ta(uint32_t tmem_d, uint32_t tmem_a, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(tmem_d),
      "r"(tmem_a), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// bounded wait that also gives up once another thread of the CTA gave up
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, int* status, volatile int* abort) {
  const uint32_t addr = smem_addr(bar);
  unsigned long long t0 = 0;
  for (uint32_t it = 0;; ++it) {
    uint32_t done;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(done)
        : "r"(addr), "r"(parity)
        : "memory");
    if (done) return true;
    if ((it & 63u) == 63u) {
      if (*abort) return false;
      const unsigned long long now = global_timer_ns();
      if (t0 == 0) {
        t0 = now;
      } else if (now - t0 > kWaitLimitNs) {
        set_status(status, kStatusTimeout);
        *abort = 1;
        return false;
      }
    }
  }
}

// non-blocking test of the phase of `parity`
__device__ __forceinline__ bool test_bar(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(done)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return done != 0;
}

// 16 lanes x 256 bits, 8 repetitions along the columns: thread t gets, per 8-column
// group g, lane t / 4 columns 8 g + 2 (t mod 4) + {0, 1}, then lane t / 4 + 8 the same
__device__ __forceinline__ void tmem_ld_16x256b_x8(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.16x256b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  tmem_wait_ld32(r);
}
__device__ __forceinline__ void tmem_st_16x256b_x8(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x256b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]),
      "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]),
      "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
// 16 lanes x 128 bits, 8 repetitions: thread t gets, per 4-column group j, column
// 4 j + (t mod 4) of lane t / 4, then of lane t / 4 + 8
__device__ __forceinline__ void tmem_st_16x128b_x8(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x128b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

constexpr float kLazyRescale = 8.f;  // log2 units; P <= 2^8 between rescales

// one 64-token x 64-dim box of a head of the cache (3-D map [rows, heads, 128], 128-byte swizzle)
__device__ __forceinline__ void tma_load_cache(void* dst, const CUtensorMap* map, int x, int head, int row,
                                               uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];" ::"r"(smem_addr(dst)),
      "l"(map), "r"(x), "r"(head), "r"(row), "r"(smem_addr(bar))
      : "memory");
}

__global__ void __launch_bounds__(kThreadsTc, 2) attn_tc_kernel(const AttnArgs p) {
  extern __shared__ __align__(1024) unsigned char smem[];
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int h = blockIdx.y;
  const int H = p.n_heads;

  pdl_launch_dependents();
  pdl_wait();
  if ((smem_addr(smem) & 1023u) != 0u) {  // the swizzled operands need a 1024-byte aligned base
    if (tid == 0) set_status(p.status, kStatusDeviceArg);
    return;
  }
  // Start-up is a chain of dependent global loads (vehicle, offsets, queries, own rows),
  // each at the latency of a loaded memory system. The batched tick hands every CTA row
  // its schedule entry (vehicle, first cache row, length: one load); the copies of the
  // vehicle's queries and own keys / values are then in flight while the rest is read.
  const __nv_bfloat16* kc;
  const __nv_bfloat16* vc;
  if (p.targs != nullptr) {
    kc = static_cast<const __nv_bfloat16*>(p.targs->k_cache[p.layer]);
    vc = static_cast<const __nv_bfloat16*>(p.targs->v_cache[p.layer]);
  } else {
    kc = static_cast<const __nv_bfloat16*>(p.k_cache);
    vc = static_cast<const __nv_bfloat16*>(p.v_cache);
  }
  AttnPlan plan_z{0, 0, 0};
  if (p.plan != nullptr) plan_z = p.plan[blockIdx.z];
  const int b = p.plan != nullptr ? plan_z.b : (p.order != nullptr ? p.order[blockIdx.z] : static_cast<int>(blockIdx.z));

  unsigned char* qt = smem + kOffQ;
  unsigned char* kslot = smem + kOffK;
  unsigned char* vslot = smem + kOffV;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint64_t* kfull = bars + 0;    // [3] K rows of a chunk staged
  uint64_t* kempty = bars + 3;   // [3] S done with a K slot
  uint64_t* vfull = bars + 6;    // [3] V rows staged
  uint64_t* vempty = bars + 9;   // [3] P V done with a V slot
  uint64_t* sfull = bars + 12;   // [2] S of a chunk in tensor memory
  uint64_t* pfull = bars + 14;   // [2] P of a chunk written over its S
  uint64_t* pvdone = bars + 16;  // [2] P V of a chunk done (one per buffer)
  uint64_t* drain = bars + 18;   // every MMA of the CTA done
  uint64_t* ktma = bars + 19;    // [3] a whole cache chunk's K rows landed by TMA
  uint64_t* vtma = bars + 22;    // [3] the same for V
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + kNumBars);
  volatile int* abort = reinterpret_cast<volatile int*>(tmem_slot + 1);

  // ---- producers' staging of chunk i (own rows fp16, cache rows bf16 converted later)
  const bool is_prod = warp >= kProdWarp0;
  const bool is_v = warp >= kProdWarp0 + 2;
  const int pt = (warp & 1) * 32 + lane;  // thread within the tensor's two warps
  const int pu = pt & 15;                 // 16-byte unit of a 256-byte row
  const int pr0 = pt >> 4;                // rows pr0, pr0 + 4, ...
  const size_t tok = static_cast<size_t>(H) * kD;
  const __half* obase = (is_v ? p.v_own : p.k_own) + static_cast<size_t>(b) * p.n_own * p.own_stride + h * kD + pu * 8;
  const __nv_bfloat16* cbase = nullptr;  // this CTA's first cache row of the tensor, set below
  long long L = 0;
  long long row0 = 0;                    // this CTA's first cache row, set below
  unsigned char* pslots = is_v ? vslot : kslot;
  // Whole cache chunks (every cache chunk but a short last one) come by two TMA box loads
  // issued by one thread of the tensor's warps (when the batched tick supplies the cache
  // maps); the own keys and a short last chunk by 16-byte copies of every thread.
  const CUtensorMap* tmap =
      (p.cache_maps != nullptr && p.targs != nullptr) ? p.cache_maps + 2 * p.layer + (is_v ? 1 : 0) : nullptr;
  uint64_t* tbar = is_v ? vtma : ktma;
  auto by_tma = [&](int i) { return tmap != nullptr && i >= 1 && static_cast<long long>(i) * kSlotKeys <= L; };
  // chunks 1 .. L / 64 are the TMA chunks, so slot s = i mod 3 sees them in order from its
  // first one (i = 3 for slot 0): the phase of chunk i on its slot's barrier
  auto tma_parity = [](int i) { return static_cast<uint32_t>((i / kSlots - (i % kSlots == 0 ? 1 : 0)) & 1); };
  auto chunk_rows = [&](int i) {
    return i == 0 ? p.n_own
                  : static_cast<int>(min(static_cast<long long>(kSlotKeys), L - (i - 1) * static_cast<long long>(kSlotKeys)));
  };
  auto issue = [&](int i) {
    unsigned char* slot = pslots + (i % kSlots) * kSlotBytes;
    const int rows = chunk_rows(i);
    const long long c0 = (i - 1) * static_cast<long long>(kSlotKeys);
    if (by_tma(i)) {
      if (pt == 0) {
        uint64_t* bar = tbar + i % kSlots;
        const int y = static_cast<int>(row0 + c0);
        mbar_arrive_expect_tx(bar, kSlotBytes);
        tma_load_cache(slot, tmap, 0, h, y, bar);
        tma_load_cache(slot + kSlotBytes / 2, tmap, 64, h, y, bar);
      }
      cp_async_commit();  // an empty group keeps one group per chunk
      return;
    }
#pragma unroll 8
    for (int m = 0; m < kSlotKeys / 4; ++m) {
      const int r = pr0 + 4 * m;
      unsigned char* dst = slot + tile128_off(r, pu);
      if (r < rows) {
        const void* src = i == 0 ? static_cast<const void*>(obase + static_cast<size_t>(r) * p.own_stride)
                                 : static_cast<const void*>(cbase + static_cast<size_t>(c0 + r) * tok);
        cp_async_16(smem_addr(dst), src);
      } else {
        *reinterpret_cast<uint4*>(dst) = make_uint4(0u, 0u, 0u, 0u);  // keys past the range: finite zeros
      }
    }
    cp_async_commit();
  };
  // queries: 64 rows x 16 units, rows >= n_q zero (one copy group per thread)
  for (int i = tid; i < 64 * 16; i += kThreadsTc) {
    const int r = i >> 4;
    const int u = i & 15;
    unsigned char* dst = qt + tile128_off(r, u);
    if (r < p.n_q)
      cp_async_16(smem_addr(dst), p.q + (static_cast<size_t>(b) * p.n_q + r) * p.q_stride + h * kD + u * 8);
    else
      *reinterpret_cast<uint4*>(dst) = make_uint4(0u, 0u, 0u, 0u);
  }
  cp_async_commit();
  if (is_prod) issue(0);  // own keys / values

  long long o_lo, o_hi;
  if (p.plan != nullptr) {
    o_lo = plan_z.lo;
    o_hi = o_lo + plan_z.len;  // a length of -1 fails the check below
  } else {
    const int64_t* offs = p.targs != nullptr ? p.targs->offsets : p.offsets;
    const int64_t* starts = p.targs != nullptr ? p.targs->starts : nullptr;
    o_lo = starts != nullptr ? starts[b] : offs[b];
    o_hi = o_lo + (offs[b + 1] - offs[b]);
  }
  if (o_lo < 0 || o_hi < o_lo || o_hi > p.max_total || (o_hi > o_lo && (kc == nullptr || vc == nullptr))) {
    cp_async_wait<0>();  // the query / own-row copies land before the CTA leaves
    set_status(p.status, kStatusDeviceArg);  // never read outside the caller's cache
    return;
  }
  L = o_hi - o_lo;
  row0 = o_lo;
  const int n_chunks = 1 + static_cast<int>((L + kSlotKeys - 1) / kSlotKeys);  // chunk 0: own keys
  cbase = (is_v ? vc : kc) + (static_cast<size_t>(o_lo) * H + h) * kD + pu * 8;

  if (tid == 0) {
    for (int i = 0; i < kSlots; ++i) {
      mbar_init(kfull + i, kProdThreads);
      mbar_init(kempty + i, 1);
      mbar_init(vfull + i, kProdThreads);
      mbar_init(vempty + i, 1);
      mbar_arrive(kempty + i);  // release 0 of every slot: free from the start
      mbar_arrive(vempty + i);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(sfull + i, 1);
      mbar_init(pfull + i, kSoftmaxWarps * 32);
      mbar_init(pvdone + i, 1);
    }
    mbar_init(drain, 1);
    // a kernel before this one has already abandoned the tick: this CTA stops below
    *abort = *reinterpret_cast<volatile int*>(p.status) != 0 ? 1 : 0;
  }
  if (warp == kMmaWarp) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (is_prod) {  // the first cache chunk; then wait for this thread's query copies
    if (pt == 0 && tmap != nullptr) {  // the TMA barriers, before the first TMA chunk; read after the CTA barrier
      for (int i = 0; i < kSlots; ++i) mbar_init(tbar + i, 1);
      fence_proxy_async();
    }
    if (n_chunks > 1) {
      issue(1);
      cp_async_wait<2>();
    } else {
      cp_async_wait<1>();
    }
  } else {
    cp_async_wait<0>();
  }
  fence_proxy_async();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(tmem_slot);
  if (*abort) {  // the tick was abandoned before this kernel: no MMA was issued
    cp_async_wait<0>();
    if (is_prod && pt == 0 && n_chunks > 1 && by_tma(1)) mbar_wait(tbar + 1, 0, p.status);  // chunk 1 landed
    if (warp == kMmaWarp)
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    return;
  }

  if (warp == kMmaWarp) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t id_s = idesc_f16_mn(64, kSlotKeys, false);
      const uint32_t id_pv_own = idesc_f16_mn(64, kD, true);       // fp16 P, fp16 own V
      const uint32_t id_pv = idesc_f16_mn(64, kD, true) | (1u << 7) | (1u << 10);  // bf16 P, bf16 cache V
      const uint32_t aq = smem_addr(qt);
      auto issue_s = [&](int i) {  // S of chunk i into buffer i & 1
        const uint32_t d = tmem + kColS + (i & 1) * kSlotKeys;
        const uint32_t kb = smem_addr(kslot + (i % kSlots) * kSlotBytes);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (kk >> 2) * 8192 + (kk & 3) * 32;
          umma_f16(d, sw128_desc(aq + off), sw128_desc(kb + off), id_s, kk > 0 ? 1u : 0u);
        }
        umma_commit(kempty + (i % kSlots));
        umma_commit(sfull + (i & 1));
      };
      auto issue_pv = [&](int i) {  // O (+)= P V of chunk i, P from tensor memory
        const uint32_t pa = tmem + kColS + (i & 1) * kSlotKeys;
        const uint32_t vb = smem_addr(vslot + (i % kSlots) * kSlotBytes);
        const uint32_t idv = i == 0 ? id_pv_own : id_pv;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {  // 16 keys = 8 columns of packed fp16 pairs
          const uint64_t bd = sw128_desc_mn(vb + kk * 2048, 8192, 1024);
          umma_f16_ta(tmem + kColO, pa + kk * 8, bd, idv, (i > 0 || kk > 0) ? 1u : 0u);  // P_hi
          umma_f16_ta(tmem + kColO, pa + kSlotKeys / 2 + kk * 8, bd, idv, 1u);          // P_lo
        }
        umma_commit(vempty + (i % kSlots));
        umma_commit(pvdone + (i & 1));
      };
      // S(ns) and P V(npv) are issued as soon as their inputs are ready: S(ns) needs
      // its K rows and P V(ns - 2) done with the buffer it overwrites, P V(npv) needs
      // P(npv) and its V rows. Each test is at most one phase behind its barrier.
      int ns = 0, npv = 0;
      unsigned long long t_idle = 0;
      for (uint32_t it = 0; npv < n_chunks; ++it) {
        bool progressed = false;
        if (ns < n_chunks && (ns < 2 || npv >= ns - 1) && test_bar(kfull + (ns % kSlots), (ns / kSlots) & 1) &&
            (ns < 2 || test_bar(pvdone + (ns & 1), ((ns - 2) >> 1) & 1))) {
          tc_fence_after();
          issue_s(ns);
          ++ns;
          progressed = true;
        }
        if (npv < ns && test_bar(pfull + (npv & 1), (npv >> 1) & 1) &&
            test_bar(vfull + (npv % kSlots), (npv / kSlots) & 1)) {
          tc_fence_after();
          issue_pv(npv);
          ++npv;
          progressed = true;
        }
        if (progressed) {
          t_idle = 0;
        } else if ((it & 63u) == 63u) {
          if (*abort) break;
          const unsigned long long now = global_timer_ns();
          if (t_idle == 0) {
            t_idle = now;
          } else if (now - t_idle > kWaitLimitNs) {
            set_status(p.status, kStatusTimeout);
            *abort = 1;
            break;
          }
        }
      }
      umma_commit(drain);  // completes once every MMA issued above has (waited on even after an abort)
      mbar_wait(drain, 0, p.status);
    }
    __syncwarp();
  } else if (is_prod) {
    // ---------------------------------------------------------------- producers
    // per chunk i: wait for its rows, convert cache rows bf16 -> fp16 in place (each
    // thread the units it copied), signal, then refill the slot of chunk i - 1 with
    // chunk i + 2 once the MMAs released it
    uint64_t* full = is_v ? vfull : kfull;
    uint64_t* empty = is_v ? vempty : kempty;
    bool ok = true;
    int issued = n_chunks > 1 ? 2 : 1;  // chunks whose loads were issued
    int i = 0;
    for (; ok && i < n_chunks; ++i) {
      if (i + 1 < n_chunks) cp_async_wait<1>();
      else cp_async_wait<0>();
      if (by_tma(i)) {
        ok = wait_bar(tbar + i % kSlots, tma_parity(i), p.status, abort);
        if (!ok) break;
      }
      // refill first when the slot of chunk i - 1 is already free (the warp agrees on it)
      bool refilled = false;
      if (i + 2 < n_chunks) {
        refilled = __all_sync(0xffffffffu, test_bar(empty + ((i + 2) % kSlots), ((i + 2) / kSlots) & 1));
        if (refilled) {
          issue(i + 2);
          issued = i + 3;
        }
      }
      if (i > 0 && !is_v) {  // cache K rows -> fp16 (V stays bf16): every read before the first write
        unsigned char* slot = pslots + (i % kSlots) * kSlotBytes;
        uint4 v[kSlotKeys / 4];
#pragma unroll
        for (int m = 0; m < kSlotKeys / 4; ++m) v[m] = *reinterpret_cast<const uint4*>(slot + tile128_off(pr0 + 4 * m, pu));
#pragma unroll
        for (int m = 0; m < kSlotKeys / 4; ++m)
          *reinterpret_cast<uint4*>(slot + tile128_off(pr0 + 4 * m, pu)) =
              make_uint4(bf16x2_to_half2(v[m].x), bf16x2_to_half2(v[m].y), bf16x2_to_half2(v[m].z),
                         bf16x2_to_half2(v[m].w));
      }
      fence_proxy_async();
      mbar_arrive(full + (i % kSlots));
      if (i + 2 < n_chunks && !refilled) {
        ok = wait_bar(empty + ((i + 2) % kSlots), ((i + 2) / kSlots) & 1, p.status, abort);
        if (ok) {
          issue(i + 2);
          issued = i + 3;
        }
      }
    }
    cp_async_wait<0>();
    // after an abort: the TMA chunks issued but not consumed land before the CTA leaves
    if (pt == 0)
      for (int j = i; j < issued; ++j)
        if (by_tma(j)) mbar_wait(tbar + j % kSlots, tma_parity(j), p.status);
  } else {
    // ---------------------------------------------------------------- softmax rows
    // Warp w owns query rows 16 w .. 16 w + 15 (tensor-memory lanes 32 w .. + 15).
    // With the 16x256b load shape each thread holds rows ra = 16 w + t / 4 and
    // rb = ra + 8, and the key pairs 8 g + 2 (t mod 4) + {0, 1} of every 8-key group
    // g; a row's maximum and sum are completed across the 4 threads of a quad. Its
    // P pairs are exactly the packed columns 4 g + (t mod 4) that the 16x128b store
    // shape gives the same thread.
    const int t4 = lane & 3;
    const int ra = warp * 16 + (lane >> 2);
    const int rbw = ra + 8;
    const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
    const float scale_log2 = 1.4426950408889634f * rsqrtf(static_cast<float>(kD));
    float m_run[2] = {-CUDART_INF_F, -CUDART_INF_F};
    float l_run[2] = {0.f, 0.f};
    bool ok = true;
    for (int i = 0; i < n_chunks; ++i) {
      const int valid = chunk_rows(i);
      ok = wait_bar(sfull + (i & 1), (i >> 1) & 1, p.status, abort);
      if (!ok) break;
      tc_fence_after();
      const uint32_t sbuf = tmem + lane_base + kColS + (i & 1) * kSlotKeys;
      uint32_t sv[32];  // [g][row a: 2 keys, row b: 2 keys]
      tmem_ld_16x256b_x8(sbuf, sv);
      float s[2][16];   // [row][g * 2 + e] for key 8 g + 2 t4 + e
#pragma unroll
      for (int g = 0; g < 8; ++g)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          s[0][2 * g + e] = __uint_as_float(sv[4 * g + e]);
          s[1][2 * g + e] = __uint_as_float(sv[4 * g + 2 + e]);
        }
      if (valid < kSlotKeys) {
#pragma unroll
        for (int g = 0; g < 8; ++g)
#pragma unroll
          for (int e = 0; e < 2; ++e)
            if (8 * g + 2 * t4 + e >= valid) {
              s[0][2 * g + e] = -CUDART_INF_F;
              s[1][2 * g + e] = -CUDART_INF_F;
            }
      }
      float mx[2], alpha[2] = {1.f, 1.f};
      bool grow = false;
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        float m4[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) m4[e] = fmaxf(fmaxf(s[r][e], s[r][e + 4]), fmaxf(s[r][e + 8], s[r][e + 12]));
        mx[r] = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
        mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
        mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
        mx[r] *= scale_log2;
        grow = grow || mx[r] > m_run[r] + kLazyRescale;
      }
      const bool any_grow = __any_sync(0xffffffffu, grow);
      if (any_grow) {
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const float m_new = fmaxf(m_run[r], mx[r]);
          alpha[r] = ex2_approx(m_run[r] - m_new);  // 0 for the first chunk
          m_run[r] = m_new;
        }
      }
      uint32_t ph[16], pl[16];  // 16x128b order: [g][row a, row b]
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const float nm = -m_run[r];
        float r4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int g = 0; g < 8; ++g) {
          const float p0 = ex2_approx(fmaf(s[r][2 * g], scale_log2, nm));
          const float p1 = ex2_approx(fmaf(s[r][2 * g + 1], scale_log2, nm));
          r4[g & 3] += p0 + p1;
          uint32_t hi, lo;
          if (i == 0) {  // own chunk: fp16 like its V rows
            hi = pack_half2(p0, p1);
            const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&hi));
            lo = pack_half2(p0 - f.x, p1 - f.y);
          } else {  // cache chunks: bf16 like the V rows
            hi = pack_bf16x2(p0, p1);
            lo = pack_bf16x2(p0 - __uint_as_float(hi << 16), p1 - __uint_as_float(hi & 0xffff0000u));
          }
          ph[2 * g + r] = hi;
          pl[2 * g + r] = lo;
        }
        float rs = (r4[0] + r4[1]) + (r4[2] + r4[3]);
        rs += __shfl_xor_sync(0xffffffffu, rs, 1);
        rs += __shfl_xor_sync(0xffffffffu, rs, 2);
        l_run[r] = l_run[r] * alpha[r] + rs;
      }
      if (any_grow && i > 0) {
        // rescale this warp's O rows once P V of the previous chunk is done
        ok = wait_bar(pvdone + ((i - 1) & 1), ((i - 1) >> 1) & 1, p.status, abort);
        if (!ok) break;
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < kD; c += 64) {
          uint32_t o[32];
          tmem_ld_16x256b_x8(tmem + lane_base + kColO + c, o);
#pragma unroll
          for (int g = 0; g < 8; ++g)
#pragma unroll
            for (int e = 0; e < 4; ++e) o[4 * g + e] = __float_as_uint(__uint_as_float(o[4 * g + e]) * alpha[e >> 1]);
          tmem_st_16x256b_x8(tmem + lane_base + kColO + c, o);
        }
      }
      // P = P_hi + P_lo over the S it came from: P_hi in columns 0..31, P_lo in 32..63
      tmem_st_16x128b_x8(sbuf, ph);
      tmem_st_16x128b_x8(sbuf + kSlotKeys / 2, pl);
      asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
      tc_fence_before();
      mbar_arrive(pfull + (i & 1));
    }
    if (ok && wait_bar(drain, 0, p.status, abort)) {  // every P V done
      tc_fence_after();
      const float inv[2] = {l_run[0] > 0.f ? 1.f / l_run[0] : 0.f, l_run[1] > 0.f ? 1.f / l_run[1] : 0.f};
      const bool va = ra < p.n_q;
      const bool vb = rbw < p.n_q;
      // A cache key beyond the fp16 range became an infinity here; where it raised a
      // score to +inf (or NaN) the row's sum is NaN: report it, the tick is abandoned.
      // (A key whose scores all fell to -inf carries weight 0, as the exact value would.)
      if ((va && !(l_run[0] == l_run[0])) || (vb && !(l_run[1] == l_run[1]))) set_status(p.status, kStatusRange);
      __half* oa = p.out + (static_cast<size_t>(b) * p.n_q + (va ? ra : 0)) * p.out_stride + h * kD + 2 * t4;
      __half* ob = p.out + (static_cast<size_t>(b) * p.n_q + (vb ? rbw : 0)) * p.out_stride + h * kD + 2 * t4;
#pragma unroll 1
      for (int c = 0; c < kD; c += 64) {
        uint32_t o[32];
        tmem_ld_16x256b_x8(tmem + lane_base + kColO + c, o);
#pragma unroll
        for (int g = 0; g < 8; ++g) {
          if (va) *reinterpret_cast<uint32_t*>(oa + c + 8 * g) =
              pack_half2(__uint_as_float(o[4 * g]) * inv[0], __uint_as_float(o[4 * g + 1]) * inv[0]);
          if (vb) *reinterpret_cast<uint32_t*>(ob + c + 8 * g) =
              pack_half2(__uint_as_float(o[4 * g + 2]) * inv[1], __uint_as_float(o[4 * g + 3]) * inv[1]);
        }
      }
      if (p.lse != nullptr && t4 == 0) {
        float* lrow = p.lse + (static_cast<size_t>(b) * H + h) * p.n_q;
        if (va) lrow[ra] = l_run[0] > 0.f ? (m_run[0] + log2f(l_run[0])) * 0.6931471805599453f : -CUDART_INF_F;
        if (vb) lrow[rbw] = l_run[1] > 0.f ? (m_run[1] + log2f(l_run[1])) * 0.6931471805599453f : -CUDART_INF_F;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

}  // namespace

bool attention_tc_eligible(const AttnArgs& a, int cache_dtype) {
  return cache_dtype == 1 && a.n_splits == 1 && a.n_q >= 1 && a.n_q <= 48 && a.n_own >= 1 && a.n_own <= kSlotKeys;
}

cudaError_t attention_tc_set_attributes() {
  return cudaFuncSetAttribute(reinterpret_cast<const void*>(&attn_tc_kernel), cudaFuncAttributeMaxDynamicSharedMemorySize,
                              kSmemTc);
}

cudaError_t launch_attention_tc(const AttnArgs& a_in, int B, cudaStream_t stream, bool pdl) {
  AttnArgs a = a_in;
  void* kargs[] = {&a};
  return launch_ex(reinterpret_cast<const void*>(&attn_tc_kernel), dim3(1, a.n_heads, B), dim3(kThreadsTc), kSmemTc,
                   stream, pdl, kargs);
}

}  // namespace fsx
