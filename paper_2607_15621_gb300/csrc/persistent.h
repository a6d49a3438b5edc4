// Launch interface of the persistent single-vehicle tick (tick_persistent.cu).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.h"

namespace fsx {

constexpr int kPersistThreads = 256;
constexpr int kPersistCluster = 4;       // CTAs per head cluster
constexpr int kPersistChunk = 16384;     // bytes per streamed weight chunk / ring slot
constexpr int kPersistSlots = 6;         // ring depth
constexpr int kPersistAChunks = 8;       // per CTA and layer: 6 QKV blocks + 2 W_o chunks
constexpr int kPersistBChunks = 3;       // per SwiGLU CTA and layer: 2 gate/up blocks + 1 W_d chunk

struct PersistArgs {
  const unsigned char* warena;  // stream-ordered fp16 weight chunks
  long long layer_bytes;        // bytes of one layer in warena
  long long a_cta_bytes;        // phase-A bytes per CTA (8 chunks)
  long long b_offset;           // offset of the phase-B part inside a layer
  long long b_cta_bytes;        // phase-B bytes per SwiGLU CTA (3 chunks)
  const float* act_emb;
  const float* pos_emb;
  const float* final_norm;
  const float* head_w;
  const float* head_b;
  const TickArgs* targs;
  int n_layers, d, H, F, n_action, n_frame, n_waypoints;
  int n_b_clusters;             // F / 64
  int frame_dtype;
  long long max_total;
  float* X;                     // [3][48][d] rotating residual buffers
  int* counters;                // [2 n_layers + 1], zeroed before every launch
  int* status;
  __half* attn_capture;         // optional [n_layers][T][H*128]
  int head;                     // 1: CTA 0 runs the single-layer waypoint head; 0: a later launch does
  unsigned long long wait_limit_ns;  // limit of the device-wide counter waits (1 s unless a test lowers it)
};

size_t persistent_smem_bytes(int d);
cudaError_t persistent_set_attributes(int d);
int persistent_max_clusters(int d, int cache_dtype);
cudaError_t launch_persistent(const PersistArgs& a, int cache_dtype, cudaStream_t stream);

}  // namespace fsx
