// Token assembly and waypoint head of the action expert (Sec. 3.1).
//
// embed: x_b = [E_act ; F_b] + P_pos into the fp32 residual stream; block 0
//        also checks the cache ranges (offsets non-decreasing; the rows of every
//        vehicle, at offsets[b] or at its optional start row, within capacity) and
//        raises the device status word, which turns the rest of the tick
//        into no-ops. Block b < B also ranks vehicle b by cache length, so the
//        attention launches can start the longest caches first (a schedule
//        only: every (vehicle, head) computes the same result in any order).
// head:  waypoint j of vehicle b = W_h RMSNorm(x_{b,j}; g_f) + b_h, fp32.
#include "device_util.cuh"
#include "kernels.h"

namespace fsx {

namespace {

__global__ void embed_kernel(const EmbedArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const int T = a.n_action + a.n_frame;
  const int row = blockIdx.x;  // b * T + t
  const int b = row / T;
  const int t = row - b * T;
  if (row == 0 && threadIdx.x == 0) {
    const int64_t* off = a.targs->offsets;
    const int64_t* st = a.targs->starts;
    bool ok = off[0] >= 0;
    for (int i = 0; i < a.B && ok; ++i) ok = off[i + 1] >= off[i];
    if (st == nullptr)
      ok = ok && off[a.B] <= a.max_total;
    else  // every vehicle's own row range lies inside the caller's cache
      for (int i = 0; i < a.B && ok; ++i) ok = st[i] >= 0 && st[i] + (off[i + 1] - off[i]) <= a.max_total;
    if (!ok) set_status(a.status, kStatusDeviceArg);
  }
  __shared__ float s_part[4];
  __shared__ int s_cnt[4];
  if (a.order != nullptr && row < a.B) {  // rank of vehicle `row`: longer caches first, ties by index
    const int64_t* off = a.targs->offsets;
    const int64_t len = off[row + 1] - off[row];
    int cnt = 0;
    for (int j = threadIdx.x; j < a.B; j += blockDim.x) {
      const int64_t lj = off[j + 1] - off[j];
      cnt += (lj > len || (lj == len && j < row)) ? 1 : 0;
    }
    for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
    if ((threadIdx.x & 31) == 0) s_cnt[threadIdx.x >> 5] = cnt;
    __syncthreads();
    if (threadIdx.x == 0) {
      int r = 0;
      for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) r += s_cnt[w];
      a.order[r] = row;
      if (a.plan != nullptr) {
        AttnPlan e;
        e.lo = a.targs->starts != nullptr ? a.targs->starts[row] : off[row];
        e.b = row;
        e.len = (len >= 0 && len <= 0x7fffffff) ? static_cast<int>(len) : -1;
        a.plan[r] = e;
      }
    }
  }
  float* xr = a.x + static_cast<size_t>(row) * a.d;
  const float* pos = a.pos_emb + static_cast<size_t>(t) * a.d;
  for (int c = threadIdx.x; c < a.d; c += blockDim.x) {
    float v;
    if (t < a.n_action) {
      v = a.act_emb[static_cast<size_t>(t) * a.d + c];
    } else {
      const size_t idx = (static_cast<size_t>(b) * a.n_frame + (t - a.n_action)) * a.d + c;
      if (a.frame_dtype == 1) {
        v = __bfloat162float(static_cast<const __nv_bfloat16*>(a.targs->frames)[idx]);
      } else {
        v = static_cast<const float*>(a.targs->frames)[idx];
      }
    }
    const float xv = v + pos[c];
    xr[c] = xv;
    a.x16[static_cast<size_t>(row) * a.d + c] = __float2half_rn(xv);
    // sum of x^2 over this 128-column group (blockDim.x == 128: one group per pass)
    const float ws = warp_sum(xv * xv);
    if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = ws;
    __syncthreads();
    if (threadIdx.x == 0)
      a.ss[static_cast<size_t>(c / 128) * a.ss_stride + row] = s_part[0] + s_part[1] + s_part[2] + s_part[3];
    __syncthreads();
  }
}

// one warp per (vehicle, waypoint)
__global__ void head_kernel(const HeadArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  if (*reinterpret_cast<volatile int*>(a.status) != 0) return;
  const int b = blockIdx.x;
  const int lane = threadIdx.x & 31;
  for (int j = threadIdx.x >> 5; j < a.n_waypoints; j += blockDim.x >> 5) {
  const float* xr = a.x + (static_cast<size_t>(b) * a.T + j) * a.d;
  float ss = 0.f;
  for (int c = lane; c < a.d; c += 32) ss += xr[c] * xr[c];
  ss = warp_sum(ss);
  const float rstd = rsqrtf(ss / static_cast<float>(a.d) + 1e-6f);
  float o0 = 0.f, o1 = 0.f;
  for (int c = lane; c < a.d; c += 32) {
    const float n = xr[c] * rstd * a.final_norm[c];
    o0 += a.head_w[c] * n;
    o1 += a.head_w[a.d + c] * n;
  }
  o0 = warp_sum(o0);
  o1 = warp_sum(o1);
  if (lane == 0) {
    float* out = a.targs != nullptr ? a.targs->waypoints : a.out;
    out[(static_cast<size_t>(b) * a.n_waypoints + j) * 2 + 0] = o0 + a.head_b[0];
    out[(static_cast<size_t>(b) * a.n_waypoints + j) * 2 + 1] = o1 + a.head_b[1];
  }
  }
}

}  // namespace

cudaError_t launch_embed(const EmbedArgs& a_in, cudaStream_t stream, bool pdl) {
  EmbedArgs a = a_in;
  void* kargs[] = {&a};
  const int rows = a.B * (a.n_action + a.n_frame);
  return launch_ex(reinterpret_cast<const void*>(&embed_kernel), dim3(rows), dim3(128), 0, stream, pdl, kargs);
}

cudaError_t launch_head(const HeadArgs& a_in, cudaStream_t stream, bool pdl) {
  HeadArgs a = a_in;
  void* kargs[] = {&a};
  return launch_ex(reinterpret_cast<const void*>(&head_kernel), dim3(a.B), dim3(32 * (a.n_waypoints < 8 ? a.n_waypoints : 8)), 0, stream,
                   pdl, kargs);
}

}  // namespace fsx
