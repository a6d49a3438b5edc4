// Asynchronous fast-slow schedule on one GPU (Sec. 3.3, Fig. 1): one vehicle's expert
// ticks run on a high-priority stream against a snapshot of the backbone cache while
// the slow system's appends run behind them on a low-priority stream. The session owns
// the committed length (SnapshotLedger): an append reserves the rows after everything
// already reserved and records an event; a tick first retires the appends whose events
// have completed and reads exactly the committed rows, so it never sees a row that is
// still being written.
//
// Two schedules (the hazard between them: the single-launch tick needs all of its CTAs
// resident at once, and the append's split-K GEMMs wait on each other's CTAs):
//   FSX_SCHED_SERIAL     appends run on the tick stream; a tick waits for an append in
//                        flight (no concurrency, no hazard);
//   FSX_SCHED_CONCURRENT appends run on their own low-priority stream with every kernel
//                        free of inter-CTA waits (fsx_append_set_concurrent: no split K),
//                        so whatever SMs an append holds are released when its kernels
//                        end and the tick's CTAs always become resident.
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>
#include <vector>

#include "../../include/fsx.h"
#include "ledger.h"

namespace fsx {
void set_error_message(const char* msg);
}

namespace {

constexpr int kRing = 16;  // argument slots (offsets, destination rows) in flight

fsx_status sfail(fsx_status s, const char* msg) {
  fsx::set_error_message(msg);
  return s;
}

}  // namespace

struct fsx_session_s {
  fsx_handle tick = nullptr;
  fsx_append_handle append = nullptr;
  int mode = FSX_SCHED_SERIAL;
  int device = 0;
  int n_layers = 0;
  int n_new = 0;
  std::vector<void*> k, v;
  cudaStream_t tick_stream = nullptr, append_stream = nullptr;
  fsx::SnapshotLedger<cudaEvent_t>* ledger = nullptr;
  std::vector<cudaEvent_t> free_events;
  // arguments: one device slot per stream (tick offsets {0, L}; append offsets {0, L} and
  // destination row), rewritten in stream order before each call from a ring of pinned
  // host slots; a host slot is reused only after the copy of its last use has run
  int64_t* d_args = nullptr;   // [5]: tick offsets [0, 2), append offsets [2, 4), append destination [4]
  int64_t* h_args = nullptr;   // pinned ring: [kRing][2] tick slots, then [kRing][3] append slots
  cudaEvent_t tick_slot_ev[kRing] = {};
  cudaEvent_t app_slot_ev[kRing] = {};
  int tick_slot = 0, app_slot = 0;
  std::mutex mu;
};

namespace {

void free_session(fsx_session_s* s) {
  if (!s) return;
  cudaSetDevice(s->device);
  if (s->tick_stream) cudaStreamSynchronize(s->tick_stream);
  if (s->append_stream) cudaStreamSynchronize(s->append_stream);
  if (s->ledger) {
    while (!s->ledger->empty()) {
      s->free_events.push_back(s->ledger->oldest());
      s->ledger->poll([](cudaEvent_t) { return true; });
    }
    delete s->ledger;
  }
  for (cudaEvent_t e : s->free_events) cudaEventDestroy(e);
  for (int i = 0; i < kRing; ++i) {
    if (s->tick_slot_ev[i]) cudaEventDestroy(s->tick_slot_ev[i]);
    if (s->app_slot_ev[i]) cudaEventDestroy(s->app_slot_ev[i]);
  }
  if (s->d_args) cudaFree(s->d_args);
  if (s->h_args) cudaFreeHost(s->h_args);
  if (s->tick_stream) cudaStreamDestroy(s->tick_stream);
  if (s->append_stream && s->append_stream != s->tick_stream) cudaStreamDestroy(s->append_stream);
  delete s;
}

// retire completed appends; their events return to the free list
long long poll_committed(fsx_session_s* s) {
  return s->ledger->poll([s](cudaEvent_t e) {
    if (cudaEventQuery(e) != cudaSuccess) return false;
    s->free_events.push_back(e);
    return true;
  });
}

}  // namespace

extern "C" {

fsx_status fsx_session_create(fsx_handle tick, fsx_append_handle append, void* const* k_cache, void* const* v_cache,
                              int n_layers, int n_new, long long capacity_rows, long long committed_rows, int mode,
                              int device, fsx_session* out) {
  fsx::set_error_message("");
  if (!out) return sfail(FSX_ERR_INVALID_ARG, "out session pointer is NULL");
  *out = nullptr;
  if (!tick || !append || !k_cache || !v_cache) return sfail(FSX_ERR_INVALID_ARG, "a handle or cache array is NULL");
  if (n_layers < 1 || n_new < 1 || committed_rows < 0 || capacity_rows < committed_rows)
    return sfail(FSX_ERR_INVALID_ARG, "n_layers, n_new >= 1 and 0 <= committed_rows <= capacity_rows required");
  if (mode != FSX_SCHED_SERIAL && mode != FSX_SCHED_CONCURRENT) return sfail(FSX_ERR_INVALID_ARG, "unknown schedule");
  for (int l = 0; l < n_layers; ++l)
    if (!k_cache[l] || !v_cache[l]) return sfail(FSX_ERR_INVALID_ARG, "a cache layer pointer is NULL");
  fsx_session_s* s = new fsx_session_s();
  s->tick = tick;
  s->append = append;
  s->mode = mode;
  s->device = device;
  s->n_layers = n_layers;
  s->n_new = n_new;
  s->k.assign(k_cache, k_cache + n_layers);
  s->v.assign(v_cache, v_cache + n_layers);
  s->ledger = new fsx::SnapshotLedger<cudaEvent_t>(committed_rows, capacity_rows);
  int lo = 0, hi = 0;
  cudaError_t e = cudaSetDevice(device);
  if (e == cudaSuccess) e = cudaDeviceGetStreamPriorityRange(&lo, &hi);
  if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&s->tick_stream, cudaStreamNonBlocking, hi);
  if (e == cudaSuccess) {
    if (mode == FSX_SCHED_SERIAL)
      s->append_stream = s->tick_stream;
    else
      e = cudaStreamCreateWithPriority(&s->append_stream, cudaStreamNonBlocking, lo);
  }
  if (e == cudaSuccess) e = cudaMalloc(&s->d_args, sizeof(int64_t) * 5);
  if (e == cudaSuccess) e = cudaMallocHost(&s->h_args, sizeof(int64_t) * 5 * kRing);
  for (int i = 0; i < kRing && e == cudaSuccess; ++i) {
    e = cudaEventCreateWithFlags(&s->tick_slot_ev[i], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&s->app_slot_ev[i], cudaEventDisableTiming);
  }
  if (e != cudaSuccess) {
    free_session(s);
    return sfail(e == cudaErrorMemoryAllocation ? FSX_ERR_OOM : FSX_ERR_CUDA, cudaGetErrorString(e));
  }
  const fsx_status st = fsx_append_set_concurrent(append, mode == FSX_SCHED_CONCURRENT);
  if (st != FSX_OK) {
    free_session(s);
    return st;
  }
  *out = s;
  return FSX_OK;
}

fsx_status fsx_session_append(fsx_session s, const void* d_x_new, float* d_hidden) {
  fsx::set_error_message("");
  if (!s || !d_x_new || !d_hidden) return sfail(FSX_ERR_INVALID_ARG, "a session or buffer pointer is NULL");
  std::lock_guard<std::mutex> lock(s->mu);
  cudaError_t e = cudaSetDevice(s->device);
  if (e != cudaSuccess) return sfail(FSX_ERR_CUDA, cudaGetErrorString(e));
  poll_committed(s);
  const long long reserved_end = s->ledger->end();  // rows the new tokens attend to: everything before them
  cudaEvent_t done = nullptr;
  if (!s->free_events.empty()) {
    done = s->free_events.back();
    s->free_events.pop_back();
  } else if ((e = cudaEventCreateWithFlags(&done, cudaEventDisableTiming)) != cudaSuccess) {
    return sfail(FSX_ERR_CUDA, cudaGetErrorString(e));
  }
  const long long dst = s->ledger->reserve(s->n_new, done);
  if (dst < 0) {
    s->free_events.push_back(done);
    return sfail(FSX_ERR_INVALID_ARG, "the append would pass the cache capacity");
  }
  // argument slot: offsets {0, reserved_end} and the destination row, staged in pinned memory
  const int slot = s->app_slot;
  s->app_slot = (slot + 1) % kRing;
  e = cudaEventSynchronize(s->app_slot_ev[slot]);  // the slot's previous copy has been consumed
  int64_t* h = s->h_args + (2 * kRing + 3 * slot);
  h[0] = 0;
  h[1] = reserved_end;
  h[2] = dst;
  int64_t* d_off = s->d_args + 2;
  if (e == cudaSuccess) e = cudaMemcpyAsync(d_off, h, 3 * sizeof(int64_t), cudaMemcpyHostToDevice, s->append_stream);
  if (e != cudaSuccess) return sfail(FSX_ERR_CUDA, cudaGetErrorString(e));
  fsx_status st = fsx_append(s->append, s->k.data(), s->v.data(), d_off, d_off + 2, 1, d_x_new, d_hidden,
                             s->append_stream);
  if (st != FSX_OK) return st;
  e = cudaEventRecord(done, s->append_stream);
  if (e == cudaSuccess) e = cudaEventRecord(s->app_slot_ev[slot], s->append_stream);
  if (e != cudaSuccess) return sfail(FSX_ERR_CUDA, cudaGetErrorString(e));
  return FSX_OK;
}

fsx_status fsx_session_tick(fsx_session s, const void* d_frames, float* d_waypoints, long long* snapshot_rows) {
  fsx::set_error_message("");
  if (!s || !d_frames || !d_waypoints) return sfail(FSX_ERR_INVALID_ARG, "a session or buffer pointer is NULL");
  std::lock_guard<std::mutex> lock(s->mu);
  cudaError_t e = cudaSetDevice(s->device);
  if (e != cudaSuccess) return sfail(FSX_ERR_CUDA, cudaGetErrorString(e));
  // the snapshot: rows of every append that has completed; in the serial schedule the
  // tick stream holds the appends in flight, so the tick reads everything reserved
  const long long L = s->mode == FSX_SCHED_SERIAL ? s->ledger->end() : poll_committed(s);
  const int slot = s->tick_slot;
  s->tick_slot = (slot + 1) % kRing;
  e = cudaEventSynchronize(s->tick_slot_ev[slot]);
  int64_t* h = s->h_args + 2 * slot;
  h[0] = 0;
  h[1] = L;
  int64_t* d_off = s->d_args;
  if (e == cudaSuccess) e = cudaMemcpyAsync(d_off, h, 2 * sizeof(int64_t), cudaMemcpyHostToDevice, s->tick_stream);
  if (e != cudaSuccess) return sfail(FSX_ERR_CUDA, cudaGetErrorString(e));
  fsx_status st = fsx_tick(s->tick, s->k.data(), s->v.data(), d_off, 1, d_frames, d_waypoints, s->tick_stream);
  if (st != FSX_OK) return st;
  if ((e = cudaEventRecord(s->tick_slot_ev[slot], s->tick_stream)) != cudaSuccess)
    return sfail(FSX_ERR_CUDA, cudaGetErrorString(e));
  if (s->mode == FSX_SCHED_SERIAL) poll_committed(s);
  if (snapshot_rows) *snapshot_rows = L;
  return FSX_OK;
}

long long fsx_session_committed(fsx_session s) {
  if (!s) return -1;
  std::lock_guard<std::mutex> lock(s->mu);
  if (cudaSetDevice(s->device) != cudaSuccess) return -1;
  return poll_committed(s);
}

long long fsx_session_reserved(fsx_session s) {
  if (!s) return -1;
  std::lock_guard<std::mutex> lock(s->mu);
  return s->ledger->end();
}

void* fsx_session_tick_stream(fsx_session s) { return s ? static_cast<void*>(s->tick_stream) : nullptr; }
void* fsx_session_append_stream(fsx_session s) { return s ? static_cast<void*>(s->append_stream) : nullptr; }

fsx_status fsx_session_sync(fsx_session s) {
  if (!s) return sfail(FSX_ERR_INVALID_ARG, "session is NULL");
  std::lock_guard<std::mutex> lock(s->mu);
  cudaError_t e = cudaSetDevice(s->device);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s->append_stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s->tick_stream);
  if (e != cudaSuccess) return sfail(FSX_ERR_CUDA, cudaGetErrorString(e));
  poll_committed(s);
  return FSX_OK;
}

void fsx_session_destroy(fsx_session s) { free_session(s); }

}  // extern "C"
