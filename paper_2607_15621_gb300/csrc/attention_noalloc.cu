// fsx_attention_noalloc: the split-KV attention entry point for callers that
// may not allocate GPU memory at run time.
//
// Some deployments reserve every byte of device memory when they start (for
// example a vehicle's real-time stack, which sizes its pools once and then
// forbids cudaMalloc because an allocation can stall on a device-wide
// synchronisation or fail when memory is fragmented, and a 50 ms control tick
// cannot absorb either). Such callers also cannot hand this library a scratch
// buffer. This variant therefore keeps its scratch -- the status word and the
// per-split partial results -- in one file-scope device array that is part of
// the library image: every GPU that loads the library holds these
// kFsxNoallocScratchBytes bytes until the process exits.
//
// Rules that follow from sharing one array:
//   * every call on a device uses the same scratch, so calls whose kernels
//     overlap on the GPU (two streams, or two host threads) race and corrupt
//     each other's results; serialise them;
//   * the array keeps the previous call's contents; the status word is cleared
//     at the start of every call, the partial slots are fully rewritten;
//   * the first call on each device looks the array's device address up
//     (cudaGetSymbolAddress) with that device current; make that first call
//     before capturing any stream. The address is kept for the life of the
//     process, so it does not survive a reset of the device's context
//     (cudaDeviceReset): do not use these entry points after one;
//   * device-side argument errors (offsets that decrease or are negative) and
//     timeouts are recorded in the array's status word, not in a caller buffer:
//     fsx_attention_noalloc_status reads and clears it.
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "../../include/fsx.h"
#include "kernels.h"

namespace fsx {
void set_error_message(const char* msg);
}

namespace {

constexpr size_t kFsxNoallocScratchBytes = static_cast<size_t>(4) << 20;  // 4 MiB
constexpr size_t kStatusSlot = 256;                                       // status word, then partials
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_noalloc_scratch[kFsxNoallocScratchBytes];

std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {};

fsx_status noalloc_fail(fsx_status s, const char* msg) {
  fsx::set_error_message(msg);
  return s;
}

// Device address of the static scratch on the current device (looked up once per device).
fsx_status scratch_base(void** base) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return noalloc_fail(FSX_ERR_CUDA, "cudaGetDevice failed or device index out of range");
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || p == nullptr) return noalloc_fail(FSX_ERR_CUDA, cudaGetErrorString(e));
    g_scratch_ptr[dev] = p;
  }
  *base = g_scratch_ptr[dev];
  return FSX_OK;
}

}  // namespace

extern "C" fsx_status fsx_attention_noalloc(const void* d_q, long long q_stride, const void* d_k_own,
                                            const void* d_v_own, long long own_stride, int n_q, int n_own,
                                            const void* d_k_cache, const void* d_v_cache, int cache_dtype,
                                            const int64_t* d_offsets, int B, int n_heads, int head_dim,
                                            int n_splits, void* d_out, float* d_lse, void* stream) {
  fsx::set_error_message("");
  if (!d_q || !d_offsets || !d_out) return noalloc_fail(FSX_ERR_INVALID_ARG, "NULL pointer argument");
  if (n_own > 0 && (!d_k_own || !d_v_own)) return noalloc_fail(FSX_ERR_INVALID_ARG, "own key/value pointers are NULL");
  if (head_dim != fsx::kHeadDim) return noalloc_fail(FSX_ERR_UNSUPPORTED, "head_dim must be 128");
  if (n_q < 1 || n_q > fsx::kTokTile) return noalloc_fail(FSX_ERR_INVALID_ARG, "n_q must be in 1..48");
  if (n_own < 0 || B < 1 || n_heads < 1) return noalloc_fail(FSX_ERR_INVALID_ARG, "n_own >= 0, B >= 1, n_heads >= 1");
  if (n_splits < 1 || n_splits > fsx::kMaxSplits) return noalloc_fail(FSX_ERR_INVALID_ARG, "n_splits must be in 1..64");
  if (cache_dtype != FSX_F32 && cache_dtype != FSX_BF16) return noalloc_fail(FSX_ERR_INVALID_ARG, "bad cache_dtype");
  if (q_stride < static_cast<long long>(n_heads) * head_dim ||
      (n_own > 0 && own_stride < static_cast<long long>(n_heads) * head_dim) || (q_stride % 8) != 0 ||
      (own_stride % 8) != 0)
    return noalloc_fail(FSX_ERR_INVALID_ARG, "strides must cover n_heads*head_dim and be multiples of 8");
  const size_t need = kStatusSlot + fsx::attention_workspace_bytes(B, n_heads, n_splits);
  if (need > kFsxNoallocScratchBytes) {
    char msg[256];
    std::snprintf(msg, sizeof(msg),
                  "B=%d, n_heads=%d, n_splits=%d need %zu bytes of scratch; the static scratch holds %zu "
                  "(use fewer splits or fsx_attention with a caller buffer)",
                  B, n_heads, n_splits, need, kFsxNoallocScratchBytes);
    return noalloc_fail(FSX_ERR_INVALID_ARG, msg);
  }

  void* base = nullptr;
  const fsx_status bs = scratch_base(&base);
  if (bs != FSX_OK) return bs;
  if (fsx::attention_set_attributes() != cudaSuccess)
    return noalloc_fail(FSX_ERR_CUDA, "cudaFuncSetAttribute failed");

  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int* status = static_cast<int*>(base);
  float* part = reinterpret_cast<float*>(static_cast<unsigned char*>(base) + kStatusSlot);
  cudaError_t e = cudaMemsetAsync(status, 0, sizeof(int), st);
  if (e != cudaSuccess) return noalloc_fail(FSX_ERR_CUDA, cudaGetErrorString(e));

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
  e = fsx::launch_attention(a, B, cache_dtype, st, false);
  if (e != cudaSuccess) return noalloc_fail(FSX_ERR_CUDA, cudaGetErrorString(e));
  return FSX_OK;
}

// The device status word of the static scratch: synchronises `stream` (the stream of
// the calls to check), returns the word and clears it. Copies one int each way; no
// allocation.
extern "C" fsx_status fsx_attention_noalloc_status(void* stream) {
  fsx::set_error_message("");
  void* base = nullptr;
  const fsx_status bs = scratch_base(&base);
  if (bs != FSX_OK) return bs;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int word = 0;
  cudaError_t e = cudaMemcpyAsync(&word, base, sizeof(int), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(base, 0, sizeof(int), st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return noalloc_fail(FSX_ERR_CUDA, cudaGetErrorString(e));
  if (word == 0) return FSX_OK;
  if (word == static_cast<int>(FSX_ERR_TIMEOUT)) return noalloc_fail(FSX_ERR_TIMEOUT, "a device-side wait timed out");
  if (word == static_cast<int>(FSX_ERR_RANGE)) return noalloc_fail(FSX_ERR_RANGE, "a cache value lies outside the fp16 range");
  return noalloc_fail(FSX_ERR_DEVICE_ARG, "device-side check: cache offsets negative or decreasing");
}
