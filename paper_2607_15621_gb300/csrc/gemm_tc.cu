// Tensor-core (tcgen05 / TMEM) projection GEMMs of the expert layer (Sec. 3.1:
// W_q/W_k/W_v, W_o and the SwiGLU block) for batches of vehicles, where the
// token count M = 42 B makes them real dense contractions.
//
// D[128 weight rows, BN tokens] = W_tile[128, K] . A[BN tokens, K]^T, fp16
// operands, fp32 accumulation in tensor memory. Each CTA owns one 128-row
// weight tile and one BN-token block and walks K in 64-wide steps through a
// 4-stage shared-memory pipeline:
//   warp 0 (one lane): producer -- the weight tile arrives as one 16 KB bulk
//     copy of a pre-swizzled image (packed at fsx_create in the 128-byte
//     swizzle layout the MMA reads), the token tile by a 2-D TMA load with the
//     same swizzle (rows past M read as zeros);
//   warp 1 (one lane): issues tcgen05.mma (M=128, N=BN, K=16) x4 per stage and
//     commits each stage back to the producer;
//   all 4 warps: epilogue -- tcgen05.ld of their 32 TMEM lanes (weight rows)
//     into a token-major tile in the idle pipeline buffers, then 16-byte
//     stores: fp16 output, SwiGLU (gate rows 16j..16j+7 next to their up rows),
//     or the fp32 residual update (each element owned by one thread), which
//     also emits each token's sum of x^2 over its 128 columns.
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

constexpr int kTcThreads = 128;
constexpr int kStages = 4;
constexpr int kTileN = 128;           // weight rows per CTA (MMA M)
constexpr int kTileK = 64;            // K per stage (128 bytes of fp16: one swizzle span)
constexpr int kWTileBytes = kTileN * kTileK * 2;  // 16 KB

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_addr(dst)),
      "l"(map), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}

template <int BN>
__host__ __device__ constexpr int tc_stage_bytes() {
  return kWTileBytes + BN * kTileK * 2;
}

template <int BN>
__host__ __device__ constexpr int tc_smem_bytes() {
  return 1024 /* barriers, tmem address */ + ((BN * 4 + 1023) / 1024) * 1024 /* 1/rms */ + 1024 /* alignment slack */ +
         kStages * tc_stage_bytes<BN>();
}

template <int BN, int EPI, bool NORM>
__global__ void __launch_bounds__(kTcThreads, 1) gemm_tc_kernel(const __grid_constant__ CUtensorMap map_a,
                                                               const TcGemmArgs p) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // 1024-byte aligned stage area (the swizzle pattern repeats every 1024 bytes)
  unsigned char* base = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(base);
  uint64_t* empty = full + kStages;
  uint64_t* done = empty + kStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  float* s_rstd = reinterpret_cast<float*>(base + 1024);
  unsigned char* stages = base + 1024 + ((BN * 4 + 1023) / 1024) * 1024;  // after the 1/rms block

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int n0 = blockIdx.x * kTileN;  // first weight row
  const int m0 = blockIdx.y * BN;      // first token
  const int KT = p.K / kTileK;
  constexpr int kAbytes = BN * kTileK * 2;
  constexpr uint32_t kTmemCols = BN <= 32 ? 32 : (BN <= 64 ? 64 : (BN <= 128 ? 128 : 256));

  pdl_launch_dependents();
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    mbar_init(done, 1);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0) {  // tensor memory for the accumulator: BN fp32 columns x 128 lanes
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *reinterpret_cast<volatile uint32_t*>(tmem_slot);

  if (warp == 0) {
    // ---- producer warp (converged; lane 0 issues): weights may stream before
    // the previous kernel finished, the token tiles only after it
    const unsigned char* wtile = p.w + static_cast<size_t>(blockIdx.x) * KT * kWTileBytes;
    const int pre = KT < kStages ? KT : kStages;
    if (lane == 0) {
      for (int kt = 0; kt < pre; ++kt) {
        mbar_arrive_expect_tx(full + kt, kWTileBytes + kAbytes);
        bulk_g2s(stages + kt * tc_stage_bytes<BN>(), wtile + static_cast<size_t>(kt) * kWTileBytes, kWTileBytes,
                 full + kt);
      }
    }
    __syncwarp();
    pdl_wait();
    for (int kt = 0; kt < KT; ++kt) {
      const int s = kt % kStages;
      unsigned char* st = stages + s * tc_stage_bytes<BN>();
      if (kt >= kStages) mbar_wait(empty + s, static_cast<uint32_t>(((kt / kStages) - 1) & 1), p.status);
      if (lane == 0) {
        if (kt >= kStages) {
          mbar_arrive_expect_tx(full + s, kWTileBytes + kAbytes);
          bulk_g2s(st, wtile + static_cast<size_t>(kt) * kWTileBytes, kWTileBytes, full + s);
        }
        tma_load_2d(st + kWTileBytes, &map_a, kt * kTileK, m0, full + s);
      }
      __syncwarp();
    }
  } else if (warp == 1) {
    // ---- MMA warp (converged; lane 0 issues)
    pdl_wait();
    constexpr uint32_t idesc = idesc_f16(kTileN, BN);
    for (int kt = 0; kt < KT; ++kt) {
      const int s = kt % kStages;
      mbar_wait(full + s, static_cast<uint32_t>((kt / kStages) & 1), p.status);
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      if (lane == 0) {
        const uint32_t a_base = smem_addr(stages + s * tc_stage_bytes<BN>());
        const uint32_t b_base = a_base + kWTileBytes;
#pragma unroll
        for (int k = 0; k < kTileK / 16; ++k)
          umma_f16(tmem, sw128_desc(a_base + k * 32), sw128_desc(b_base + k * 32), idesc, (kt > 0 || k > 0) ? 1u : 0u);
        umma_commit(empty + s);
      }
      __syncwarp();
    }
    if (lane == 0) umma_commit(done);
    __syncwarp();
  }

  // ---- epilogue: every warp reads its 32 lanes (weight rows n0 + 32 warp + lane)
  pdl_wait();  // the residual stream written by the previous kernel is read below
  if (NORM) {  // 1/rms of the tile's tokens from the per-128-column partial sums of x^2
    for (int t = tid; t < BN; t += kTcThreads) {
      float ss = 0.f;
      if (m0 + t < p.M)
        for (int j = 0; j < p.n_ss; ++j) ss += __ldcg(p.ss_in + static_cast<size_t>(j) * p.ss_stride + m0 + t);
      s_rstd[t] = rsqrtf(ss / static_cast<float>(p.K) + 1e-6f);
    }
  }
  mbar_wait(done, 0, p.status);
  __syncthreads();  // 1/rms visible
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const int row = warp * 32 + lane;
  const uint32_t taddr = tmem + (static_cast<uint32_t>(warp * 32) << 16);
  // TMEM -> registers -> token-major tile in the (now idle) pipeline buffers
  constexpr int kSH = kTileN + 8;  // fp16 row stride (store)
  constexpr int kSG = 64 + 8;      // fp16 row stride (SwiGLU: 64 columns per tile)
  constexpr int kSF = kTileN + 4;  // fp32 row stride (residual)
  __half* tH = reinterpret_cast<__half*>(stages);
  float* tF = reinterpret_cast<float*>(stages);
  for (int c0 = 0; c0 < BN; c0 += 16) {
    float v[16];
    __syncwarp();  // tcgen05.ld.sync.aligned needs the whole warp converged
    tmem_ld16(taddr + static_cast<uint32_t>(c0), v);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      float val = v[j];
      if (NORM) val *= s_rstd[c0 + j];
      if (EPI == kEpiStore) {
        tH[(c0 + j) * kSH + row] = __float2half_rn(val);
      } else if (EPI == kEpiResidual) {
        tF[(c0 + j) * kSF + row] = val;
      } else {  // SwiGLU: lane l (l % 16 < 8) holds a gate row, lane l + 8 its up row
        const float up = __shfl_down_sync(0xffffffffu, val, 8);
        const __half hv = __float2half_rn(__fdividef(val, 1.f + __expf(-val)) * up);
        if ((lane & 8) == 0) tH[(c0 + j) * kSG + (row >> 4) * 8 + (lane & 7)] = hv;
      }
    }
  }
  __syncthreads();
  // coalesced 16-byte stores of the tile's token rows
  if (EPI == kEpiStore) {
    for (int i = tid; i < BN * (kTileN / 8); i += kTcThreads) {
      const int t = i / (kTileN / 8);
      const int u = i % (kTileN / 8);
      if (m0 + t < p.M)
        *reinterpret_cast<uint4*>(p.y + static_cast<size_t>(m0 + t) * p.ldy + n0 + u * 8) =
            *reinterpret_cast<const uint4*>(tH + t * kSH + u * 8);
    }
  } else if (EPI == kEpiSwiglu) {
    for (int i = tid; i < BN * 8; i += kTcThreads) {
      const int t = i >> 3;
      const int u = i & 7;
      if (m0 + t < p.M)
        *reinterpret_cast<uint4*>(p.y + static_cast<size_t>(m0 + t) * p.ldy + n0 / 2 + u * 8) =
            *reinterpret_cast<const uint4*>(tH + t * kSG + u * 8);
    }
  } else {
    // warp w handles token rows w, w+4, ...: lane = 4-column group, so a warp covers
    // one full 128-column row and reduces its x^2 partial with shuffles
    constexpr int kRows = BN / 4;
    constexpr int kBatch = kRows % 8 == 0 ? 8 : 4;  // divides kRows (12, 32 or 64)
    for (int r0 = 0; r0 < kRows; r0 += kBatch) {
      float4 a[kBatch];
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        const int t = (r0 + b) * 4 + warp;
        a[b] = m0 + t < p.M ? *reinterpret_cast<const float4*>(p.xo + static_cast<size_t>(m0 + t) * p.ldxo + n0 + lane * 4)
                            : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        const int t = (r0 + b) * 4 + warp;
        const float4 r = *reinterpret_cast<const float4*>(tF + t * kSF + lane * 4);
        const float4 x = make_float4(a[b].x + r.x, a[b].y + r.y, a[b].z + r.z, a[b].w + r.w);
        const float ss = warp_sum(x.x * x.x + x.y * x.y + x.z * x.z + x.w * x.w);
        if (m0 + t < p.M) {
          const size_t idx = static_cast<size_t>(m0 + t) * p.ldxo + n0 + lane * 4;
          *reinterpret_cast<float4*>(p.xo + idx) = x;
          uint2 pk;
          pk.x = pack_half2(x.x, x.y);
          pk.y = pack_half2(x.z, x.w);
          *reinterpret_cast<uint2*>(p.xo16 + idx) = pk;
          if (lane == 0 && p.ss_out != nullptr) p.ss_out[static_cast<size_t>(blockIdx.x) * p.ss_stride + m0 + t] = ss;
        }
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 0)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
}

template <int BN, int EPI, bool NORM>
const void* tc_fn() {
  return reinterpret_cast<const void*>(&gemm_tc_kernel<BN, EPI, NORM>);
}

const void* tc_select(int bn, int epi, bool norm, size_t* smem) {
#define FSX_TC(BN_, EPI_, NORM_)                      \
  if (bn == BN_ && epi == EPI_ && norm == NORM_) {    \
    *smem = tc_smem_bytes<BN_>();                      \
    return tc_fn<BN_, EPI_, NORM_>();                  \
  }
  FSX_TC(48, kEpiStore, true)
  FSX_TC(48, kEpiStore, false)
  FSX_TC(48, kEpiSwiglu, true)
  FSX_TC(48, kEpiResidual, false)
  FSX_TC(128, kEpiStore, true)
  FSX_TC(128, kEpiSwiglu, true)
  FSX_TC(128, kEpiResidual, false)
  FSX_TC(256, kEpiStore, true)
  FSX_TC(256, kEpiSwiglu, true)
  FSX_TC(256, kEpiResidual, false)
#undef FSX_TC
  return nullptr;
}

}  // namespace

cudaError_t gemm_tc_set_attributes() {
  const int bns[3] = {48, 128, 256};
  const int epis[3] = {kEpiStore, kEpiSwiglu, kEpiResidual};
  for (int bn : bns)
    for (int epi : epis)
      for (int norm = 0; norm < 2; ++norm) {
        size_t smem = 0;
        const void* fn = tc_select(bn, epi, norm != 0, &smem);
        if (!fn) continue;
        cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
      }
  return cudaSuccess;
}

cudaError_t launch_gemm_tc(const CUtensorMap& map_a, const TcGemmArgs& args, int bn, int epi, bool norm,
                           cudaStream_t stream, bool pdl) {
  size_t smem = 0;
  const void* fn = tc_select(bn, epi, norm, &smem);
  if (!fn || args.N % kTileN != 0 || args.K % kTileK != 0) return cudaErrorInvalidValue;
  CUtensorMap map = map_a;
  TcGemmArgs a = args;
  void* kargs[] = {&map, &a};
  const dim3 grid(args.N / kTileN, (args.M + bn - 1) / bn);
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

bool encode_act_map(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void* sym = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &sym, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || sym == nullptr)
      return false;
    fn = reinterpret_cast<EncodeTiledFn>(sym);
  }
  const cuuint64_t dims[2] = {cols, rows};
  const cuuint64_t strides[1] = {cols * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kTileK), box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace fsx
