// Weight-streaming projection GEMMs of the expert layer (Sec. 3.1: the
// rectangular W_q/W_k/W_v projections, the output projection W_o and the
// SwiGLU block), for the small token counts of a tick (M = 42 B rows).
//
// Y[M, N] = A[M, K] . W[N, K]^T on fp16 tensor cores (mma.sync m16n8k16, fp32
// accumulation) with the weights as the 16-row operand ("swap-AB"), so a
// 48-token tile is six n8 column tiles and every weight byte is used for six
// MMAs. Each CTA owns nb x 16 weight rows and a K range; its weight tile is a
// contiguous run of fragment-ordered blocks that one thread fetches with bulk
// copies (mbarrier completion) BEFORE waiting on the previous kernel, so the
// weight stream overlaps the tail of the preceding step. The activation tile
// (48 x K range, fp16) arrives by per-row bulk copies on a second mbarrier:
// for the RMSNorm-fused projections it is the fp16 copy of the residual
// stream (the norm gain is folded into the packed weights and the per-row
// 1/rms, computed from the staged tile, scales the accumulators), otherwise
// the fp16 input rows (attention output, SwiGLU activations).
// Warps split the K range; a shared-memory reduction combines them and the
// epilogue stores fp16, applies the SwiGLU gate to row pairs packed next to
// each other, or adds the split-K sum into the fp32 residual stream. The K
// splits of one output tile form a thread-block cluster: every CTA reduces
// its warps into shared memory, and after a cluster barrier each CTA sums a
// slice of the tile over all splits through distributed shared memory in
// split order, so the residual update is deterministic and needs no atomics.
#include <cooperative_groups.h>

#include "device_util.cuh"
#include "kernels.h"

namespace cg = cooperative_groups;

namespace fsx {

namespace {

constexpr int kThreads = 128;   // 4 warps
constexpr int kRedStride = kTokTile + 4;

__host__ __device__ constexpr int a_stride(int ks) { return ks + 8; }  // halves, 16-byte row pad

// Shared memory: [256 B barriers + 1/rms][weights][activation tile, reused as
// the cross-warp reduction buffer after the MMAs][split-K receive buffer].
constexpr int kRecvRows = kTokTile + 8;  // >= n_split * ceil(48 / n_split) for n_split <= 8

__host__ __device__ inline size_t gemm_a_region(int nb, int ks) {
  const size_t a = static_cast<size_t>(kTokTile) * a_stride(ks) * 2;
  const size_t r = static_cast<size_t>(4) * (16 * nb) * kRedStride * 4;
  return a > r ? a : r;
}

__host__ __device__ inline size_t gemm_smem_bytes(int nb, int ks, int epi) {
  return 256 + static_cast<size_t>(nb) * (ks / 16) * 512 + gemm_a_region(nb, ks) +
         (epi == kEpiResidual ? static_cast<size_t>(kRecvRows) * (16 * nb) * 4 : 0);
}

template <int NB, int PRO, int EPI>
__global__ void __launch_bounds__(kThreads) gemm_ws_kernel(const GemmArgs p) {
  constexpr int NT = 16 * NB;
  extern __shared__ __align__(128) unsigned char smem[];
  const int ks = p.ks;
  const int lda_s = a_stride(ks);
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem);       // weights
  uint64_t* act_bar = bar + 1;                              // activation tile
  float* s_rstd = reinterpret_cast<float*>(smem + 16);     // [48] per-row 1/rms (kProNorm)
  uint4* sW = reinterpret_cast<uint4*>(smem + 256);
  __half* sA = reinterpret_cast<__half*>(smem + 256 + static_cast<size_t>(NB) * (ks / 16) * 512);
  float* sR = reinterpret_cast<float*>(sA);  // reused once every warp finished its MMAs
  float* recv = reinterpret_cast<float*>(reinterpret_cast<unsigned char*>(sA) + gemm_a_region(NB, ks));

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int nb0 = blockIdx.x * NB;
  const int k0 = blockIdx.y * ks;
  const int kl = min(ks, p.K - k0);
  const int kb_total = p.K / 16;

  pdl_launch_dependents();
  if (tid == 0) {
    mbar_init(bar, 1);
    mbar_init(act_bar, 1);
    mbar_arrive_expect_tx(bar, static_cast<uint32_t>(NB * (kl / 16) * 512));
#pragma unroll
    for (int j = 0; j < NB; ++j) {
      const uint4* src = p.w + (static_cast<size_t>(nb0 + j) * kb_total + k0 / 16) * 32;
      bulk_g2s(sW + static_cast<size_t>(j) * (ks / 16) * 32, src, static_cast<uint32_t>((kl / 16) * 512), bar);
    }
  }
  __syncthreads();  // barriers initialised before anyone polls them
  pdl_wait();
  const bool weights_ok = mbar_wait(bar, 0, p.status);
  // A CTA of a split-K cluster never leaves early: its partners read its shared
  // memory after the cluster barrier. On a raised status it computes a result
  // the flagged tick discards; every other kernel simply returns.
  if (EPI != kEpiResidual && (!weights_ok || *reinterpret_cast<volatile int*>(p.status) != 0)) return;

  const int n_mtiles = (p.M + kTokTile - 1) / kTokTile;
  const int mt_begin = blockIdx.z * p.m_tiles_per_cta;
  const int mt_end = min(n_mtiles, mt_begin + p.m_tiles_per_cta);
  const __half* a_src = PRO == kProNorm ? p.x16 : p.a;
  const int a_ld = PRO == kProNorm ? p.ldx16 : p.lda;

  for (int mt = mt_begin; mt < mt_end; ++mt) {
    const int m0 = mt * kTokTile;
    const int rows = min(kTokTile, p.M - m0);
    // ---------------- prologue: activation rows -> sA by bulk copies, padding rows zeroed
    if (warp == 0) {
      if (lane == 0) mbar_arrive_expect_tx(act_bar, static_cast<uint32_t>(rows * kl * 2));
      __syncwarp();
      for (int r = lane; r < rows; r += 32)
        bulk_g2s(sA + static_cast<size_t>(r) * lda_s, a_src + static_cast<size_t>(m0 + r) * a_ld + k0,
                 static_cast<uint32_t>(kl * 2), act_bar);
    }
    for (int i = tid; i < (kTokTile - rows) * (kl / 8); i += kThreads) {
      const int r = rows + i / (kl / 8);
      const int c = (i % (kl / 8)) * 8;
      *reinterpret_cast<uint4*>(sA + static_cast<size_t>(r) * lda_s + c) = make_uint4(0u, 0u, 0u, 0u);
    }
    mbar_wait(act_bar, static_cast<uint32_t>((mt - mt_begin) & 1), p.status);
    if (PRO == kProNorm) {  // 1/rms of each staged row (the whole row: ks == K)
      for (int r = warp; r < kTokTile; r += 4) {
        const __half* row = sA + static_cast<size_t>(r) * lda_s;
        float ss = 0.f;
        for (int c = lane * 8; c < kl; c += 256) {
          const uint4 u = *reinterpret_cast<const uint4*>(row + c);
          const __half2* hv = reinterpret_cast<const __half2*>(&u);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 f = __half22float2(hv[e]);
            ss += f.x * f.x + f.y * f.y;
          }
        }
        ss = warp_sum(ss);
        if (lane == 0) s_rstd[r] = rsqrtf(ss / static_cast<float>(p.K) + 1e-6f);
      }
    }
    __syncthreads();

    // ---------------- tensor-core main loop: warp w takes 64-wide K groups w, w+4, ...
    float acc[NB][6][4];
#pragma unroll
    for (int j = 0; j < NB; ++j)
#pragma unroll
      for (int t = 0; t < 6; ++t)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[j][t][e] = 0.f;

    const int n_groups = kl / 64;
    for (int g = warp; g < n_groups; g += 4) {
      uint32_t bfr[6][4][2];
#pragma unroll
      for (int t = 0; t < 6; ++t) {
#pragma unroll
        for (int kp = 0; kp < 2; ++kp) {
          const __half* src = sA + static_cast<size_t>(t * 8 + (lane & 7)) * lda_s + g * 64 + kp * 32 + (lane >> 3) * 8;
          ldsm_x4(bfr[t][2 * kp][0], bfr[t][2 * kp][1], bfr[t][2 * kp + 1][0], bfr[t][2 * kp + 1][1], smem_addr(src));
        }
      }
#pragma unroll
      for (int j = 0; j < NB; ++j) {
#pragma unroll
        for (int kb = 0; kb < 4; ++kb) {
          const uint4 af = sW[(static_cast<size_t>(j) * (ks / 16) + g * 4 + kb) * 32 + lane];
#pragma unroll
          for (int t = 0; t < 6; ++t) mma_f16_16816(acc[j][t], af.x, af.y, af.z, af.w, bfr[t][kb][0], bfr[t][kb][1]);
        }
      }
    }

    __syncthreads();  // the activation tile becomes the reduction buffer
    // ---------------- cross-warp reduction through shared memory
#pragma unroll
    for (int j = 0; j < NB; ++j) {
#pragma unroll
      for (int t = 0; t < 6; ++t) {
        const int n = j * 16 + (lane >> 2);
        const int m = t * 8 + 2 * (lane & 3);
        float* r0 = sR + (static_cast<size_t>(warp) * NT + n) * kRedStride + m;
        float* r1 = r0 + 8 * kRedStride;
        *reinterpret_cast<float2*>(r0) = make_float2(acc[j][t][0], acc[j][t][1]);
        *reinterpret_cast<float2*>(r1) = make_float2(acc[j][t][2], acc[j][t][3]);
      }
    }
    __syncthreads();

    auto red = [&](int n, int m) -> float {
      const float* r = sR + static_cast<size_t>(n) * kRedStride + m;
      const float v = r[0] + r[NT * kRedStride] + r[2 * NT * kRedStride] + r[3 * NT * kRedStride];
      return PRO == kProNorm ? v * s_rstd[m] : v;
    };

    // ---------------- epilogue
    if (EPI == kEpiStore) {
      constexpr int NP = NT / 2;
      for (int i = tid; i < NP * kTokTile; i += kThreads) {
        const int n = (i % NP) * 2;
        const int m = i / NP;
        if (m0 + m < p.M) {
          const uint32_t v = pack_half2(red(n, m), red(n + 1, m));
          *reinterpret_cast<uint32_t*>(p.y + static_cast<size_t>(m0 + m) * p.ldy + nb0 * 16 + n) = v;
        }
      }
    } else if (EPI == kEpiResidual) {
      // Split-K sum over the cluster, in split order: every CTA pushes the rows
      // another rank owns into that rank's receive buffer (remote shared-memory
      // stores), one cluster barrier, then each owner adds its rows locally.
      cg::cluster_group cluster = cg::this_cluster();
      const int n_split = static_cast<int>(cluster.num_blocks());
      const int rank = static_cast<int>(cluster.block_rank());
      const int rows_per = (kTokTile + n_split - 1) / n_split;
      for (int i = tid; i < kTokTile * NT; i += kThreads) {
        const int m = i / NT;
        const int n = i - m * NT;
        const int owner = m / rows_per;
        float* dst = cluster.map_shared_rank(recv, owner);
        dst[(static_cast<size_t>(rank) * rows_per + (m - owner * rows_per)) * NT + n] = red(n, m);
      }
      cluster.sync();
      const int r0 = rank * rows_per;
      const int r1 = min(kTokTile, r0 + rows_per);
      for (int i = tid; i < (r1 - r0) * NT; i += kThreads) {
        const int mm = i / NT;
        const int n = i - mm * NT;
        const int m = r0 + mm;
        if (m0 + m < p.M) {
          float acc_s = 0.f;
          for (int sp = 0; sp < n_split; ++sp) acc_s += recv[(static_cast<size_t>(sp) * rows_per + mm) * NT + n];
          const size_t idx = static_cast<size_t>(m0 + m) * p.ldxo + nb0 * 16 + n;
          const float xn = p.xo[idx] + acc_s;
          p.xo[idx] = xn;
          p.xo16[idx] = __float2half_rn(xn);
        }
      }
      cluster.sync();  // receive buffers are refilled by the next m-tile only after every owner summed
    } else {  // kEpiSwiglu: block j rows 0..7 = gate of h columns (nb0+j)*8 + r, rows 8..15 = up
      constexpr int NH = NB * 8;
      for (int i = tid; i < NH * kTokTile; i += kThreads) {
        const int hc = i % NH;
        const int m = i / NH;
        if (m0 + m < p.M) {
          const int j = hc >> 3;
          const int r = hc & 7;
          const float g = red(j * 16 + r, m);
          const float u = red(j * 16 + 8 + r, m);
          const float hval = g / (1.f + __expf(-g)) * u;
          p.y[static_cast<size_t>(m0 + m) * p.ldy + nb0 * 8 + hc] = __float2half_rn(hval);
        }
      }
    }
    __syncthreads();  // sA / sR reused by the next m-tile
  }
}

template <int NB, int PRO, int EPI>
const void* kernel_ptr() {
  return reinterpret_cast<const void*>(&gemm_ws_kernel<NB, PRO, EPI>);
}

const void* select_kernel(int nb, int pro, int epi) {
#define FSX_SEL(NB_, PRO_, EPI_) \
  if (nb == NB_ && pro == PRO_ && epi == EPI_) return kernel_ptr<NB_, PRO_, EPI_>();
  FSX_SEL(1, kProNorm, kEpiStore)
  FSX_SEL(2, kProNorm, kEpiStore)
  FSX_SEL(3, kProNorm, kEpiStore)
  FSX_SEL(1, kProNorm, kEpiSwiglu)
  FSX_SEL(2, kProNorm, kEpiSwiglu)
  FSX_SEL(1, kProCopy, kEpiResidual)
  FSX_SEL(2, kProCopy, kEpiResidual)
  FSX_SEL(1, kProCopy, kEpiStore)
  FSX_SEL(2, kProCopy, kEpiStore)
#undef FSX_SEL
  return nullptr;
}

}  // namespace

cudaError_t gemm_set_attributes() {
  const int nbs[3] = {1, 2, 3};
  const int pros[2] = {kProNorm, kProCopy};
  const int epis[3] = {kEpiStore, kEpiResidual, kEpiSwiglu};
  for (int nb : nbs)
    for (int pro : pros)
      for (int epi : epis) {
        const void* fn = select_kernel(nb, pro, epi);
        if (!fn) continue;
        cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, 220 * 1024);
        if (e != cudaSuccess) return e;
      }
  return cudaSuccess;
}

GemmPlan plan_gemm(int n_rows, int K, int M, int nb, int ks, int prologue, int epilogue, int sm_count) {
  GemmPlan pl{};
  pl.nb = nb;
  pl.ks = ks;
  pl.prologue = prologue;
  pl.epilogue = epilogue;
  if (epilogue == kEpiResidual) {  // the K splits of a tile form one cluster (portable size <= 8)
    const int min_ks = (K + 8 * 64 - 1) / (8 * 64) * 64;
    if (ks < min_ks) ks = min_ks;
    pl.ks = ks;
  }
  const int nx = n_rows / (16 * nb);
  const int ny = (K + ks - 1) / ks;
  const int m_tiles = (M + kTokTile - 1) / kTokTile;
  int nz = (4 * sm_count) / (nx * ny);
  if (nz < 1) nz = 1;
  if (nz > m_tiles) nz = m_tiles;
  const int per = (m_tiles + nz - 1) / nz;
  nz = (m_tiles + per - 1) / per;
  pl.grid = dim3(nx, ny, nz);
  pl.smem = gemm_smem_bytes(nb, pl.ks, epilogue);
  return pl;
}

cudaError_t launch_gemm(const GemmPlan& pl, const GemmArgs& args_in, cudaStream_t stream, bool pdl) {
  GemmArgs args = args_in;
  args.ks = pl.ks;
  const int m_tiles = (args.M + kTokTile - 1) / kTokTile;
  args.m_tiles_per_cta = (m_tiles + static_cast<int>(pl.grid.z) - 1) / static_cast<int>(pl.grid.z);
  const void* fn = select_kernel(pl.nb, pl.prologue, pl.epilogue);
  if (!fn) return cudaErrorInvalidValue;
  void* kargs[] = {&args};
  const int cluster_y = pl.epilogue == kEpiResidual ? static_cast<int>(pl.grid.y) : 1;
  return launch_ex(fn, pl.grid, dim3(kThreads), pl.smem, stream, pdl, kargs, cluster_y);
}

cudaError_t launch_ex(const void* fn, dim3 grid, dim3 block, size_t smem, cudaStream_t stream, bool pdl,
                      void** args, int cluster_y, int cluster_x) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  int n = 0;
  if (pdl) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  if (cluster_y > 1 || cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = static_cast<unsigned>(cluster_x);
    attr[n].val.clusterDim.y = static_cast<unsigned>(cluster_y);
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelExC(&cfg, fn, args);
}

}  // namespace fsx
