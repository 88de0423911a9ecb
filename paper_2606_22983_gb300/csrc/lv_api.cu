// C-ABI entry points of liblv (see include/lv.h): argument checks, device
// metadata, staging of host-pointer arguments, and kernel launches.
#include <algorithm>
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <new>
#include <deque>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "lv_internal.cuh"

// One NVTX range per entry point, so that a profiler's timeline shows which liblv call
// launched which kernels (no cost without a tool attached).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// Pages or slots touched by transfers that may still be running: a byte per
// index for lookups, and the list of marked indices for clearing.
struct MarkSet {
  std::vector<uint8_t> on;
  std::vector<int32_t> list;
  void resize(int64_t n) { on.assign((size_t)(n > 0 ? n : 1), 0); }
  void add(int32_t x) {
    if (x >= 0 && (size_t)x < on.size() && !on[x]) {
      on[x] = 1;
      list.push_back(x);
    }
  }
  bool has(int32_t x) const { return x < 0 || (size_t)x >= on.size() || on[x] != 0; }
  void clear() {
    for (int32_t x : list) on[x] = 0;
    list.clear();
  }
};

struct lv_pool {
  lv::DevPool d{};
  int device = 0;
  int num_sms = 0;
  int32_t epoch = 0;
  int exchange_ctas = 0;           // grid of the exchange copy kernel
  int remap_per_thread = 0;        // entries per thread of k_remap (0: by batch size)
  unsigned char* sched_scratch = nullptr;   // lv_schedule's keys and costs
  lv::ResidentScratch rs{};        // lv_make_resident / lv_turn buffers
  // LV_RESIDENT_ASYNC_COPY: the copies run on s_copy; consecutive steps alternate
  // between two task lists and control-word sets (rs_alt shares everything else)
  lv::ResidentScratch rs_alt{};
  uint32_t rs_seq = 0;
  cudaStream_t s_copy = nullptr;
  cudaEvent_t ev_planned = nullptr;
  cudaEvent_t ev_copy_start = nullptr, ev_copy_end = nullptr;
  cudaEvent_t ev_copied[2] = {nullptr, nullptr};
  bool copied_pending[2] = {false, false};   // an async copy used scratch set b
  // LV_MODE_STAGED | LV_MODE_ASYNC: unpacks on s_unpack; the last call's D2H, H2D and
  // unpack completions (each next call's transfers wait on them) and its whole end
  cudaStream_t s_unpack = nullptr;
  cudaEvent_t ev_st_d2h = nullptr, ev_st_h2d = nullptr, ev_st_unpack = nullptr,
              ev_st_packed = nullptr, ev_st_done = nullptr;
  bool st_pending = false;
  // what those calls touch while they may still run: pages their unpacks write, slots
  // their D2H copies write, slots their H2D copies read; a new call waits for an event
  // only when it touches a marked page or slot
  MarkSet st_loaded, st_written, st_read;
  // staging runs of the staged path, used by alternate calls and kept between calls;
  // st_buf_done[b] completes when the call that last used run b has finished with it
  void* st_buf[2] = {nullptr, nullptr};
  size_t st_buf_bytes[2] = {0, 0};
  cudaEvent_t st_buf_done[2] = {nullptr, nullptr};
  bool st_buf_used[2] = {false, false};
  uint32_t st_seq = 0;
  // staged path: side streams for the copy engines, a host copy of the tasks, sync events
  cudaStream_t s_d2h = nullptr, s_h2d = nullptr;
  int4* tasks_host = nullptr;
  size_t tasks_host_cap = 0;
  std::vector<cudaEvent_t> sync_events;
  int stage_ctas = 0;
  bool stage_tma = true;           // pack/unpack with TMA bulk copies (else 16-byte LSU copies)
  int32_t fault_kind = LV_FAULT_NONE;   // lv_inject_fault: one-shot, after `fault_after` more events
  int32_t fault_after = 0;
  // copy-kernel timing (lv_timing_enable): event pairs recorded per kind, reused
  bool timing = false;
  std::vector<lv::EventPair> ev_free;
  // a deque: the pointer timing_pair returns stays valid while later pairs are added
  std::deque<lv::EventPair> ev_used[LV_TIMING_KINDS];
  bool own_host = false;
  void* host_base = nullptr;       // host-visible address of the host pool
  std::vector<void*> dev_allocs;
  cudaMemPool_t mp = nullptr;      // stream-ordered staging memory
  // device-driven steps whose kernels all run on the caller's stream go out as one
  // CUDA graph launch: one instantiated graph per shape of the launch sequence, its
  // kernel nodes' arguments replaced for every step
  struct StepGraph {
    std::vector<const void*> funcs;
    std::vector<dim3> grids, blocks;
    std::vector<size_t> smems;
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    std::vector<cudaGraphNode_t> nodes;   // kernel nodes in launch order
  };
  std::vector<StepGraph> step_graphs;
  bool step_graphs_on = true;
  cudaStream_t s_capture = nullptr;
};

namespace {

using lv::DevPool;

#define LV_TRY(expr)                              \
  do {                                            \
    cudaError_t _e = (expr);                      \
    if (_e != cudaSuccess) return lv_cuda_fail(_e); \
  } while (0)

lv_status lv_cuda_fail(cudaError_t e) {
  if (e == cudaErrorMemoryAllocation) {
    cudaGetLastError();
    return LV_ERR_OOM;
  }
  return LV_ERR_CUDA;
}

class DeviceGuard {
 public:
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev_) == cudaSuccess && prev_ != dev) {
      cudaSetDevice(dev);
      restore_ = true;
    }
  }
  ~DeviceGuard() {
    if (restore_) cudaSetDevice(prev_);
  }

 private:
  int prev_ = 0;
  bool restore_ = false;
};

bool is_device_ptr(const void* p) {
  cudaPointerAttributes a{};
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

// The address the GPU uses for p: p itself for device or managed memory, the
// device alias of mapped page-locked host memory, else nullptr (pageable memory).
const void* gpu_view(const void* p) {
  cudaPointerAttributes a{};
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return p;
  if (a.type == cudaMemoryTypeHost) return a.devicePointer;
  return nullptr;
}

// Per-call staging.  Device, managed and mapped page-locked host arguments are
// used in place (the kernels read and write page-locked host memory over the host
// link, in stream order); pageable host inputs are copied in, and pageable (or
// absent) outputs get stream-ordered device buffers that are copied back at the end.
class Staging {
 public:
  Staging(lv_pool* pool, cudaStream_t s) : pool_(pool), s_(s) {}
  ~Staging() {
    for (void* t : temps_) cudaFreeAsync(t, s_);
  }

  lv_status in(const void* user, size_t bytes, const void** dev) {
    *dev = nullptr;
    if (bytes == 0) return LV_OK;
    if (user == nullptr) return LV_ERR_INVALID;
    if (const void* v = gpu_view(user)) {
      *dev = v;
      return LV_OK;
    }
    void* t = nullptr;
    lv_status st = temp(bytes, &t);
    if (st != LV_OK) return st;
    LV_TRY(cudaMemcpyAsync(t, user, bytes, cudaMemcpyHostToDevice, s_));
    *dev = t;
    return LV_OK;
  }

  // required: a device buffer is needed even when the caller passes NULL
  lv_status out(void* user, size_t bytes, void** dev, bool required) {
    *dev = nullptr;
    if (bytes == 0) return LV_OK;
    if (user != nullptr) {
      if (const void* v = gpu_view(user)) {
        *dev = const_cast<void*>(v);
        return LV_OK;
      }
    }
    if (user == nullptr && !required) return LV_OK;
    void* t = nullptr;
    lv_status st = temp(bytes, &t);
    if (st != LV_OK) return st;
    *dev = t;
    if (user != nullptr) backs_.push_back({user, t, bytes});
    return LV_OK;
  }

  lv_status finish() {
    for (const Back& b : backs_) LV_TRY(cudaMemcpyAsync(b.user, b.dev, b.bytes, cudaMemcpyDeviceToHost, s_));
    backs_.clear();
    return LV_OK;
  }

 private:
  struct Back {
    void* user;
    void* dev;
    size_t bytes;
  };
  lv_status temp(size_t bytes, void** t) {
    cudaError_t e = cudaMallocFromPoolAsync(t, bytes, pool_->mp, s_);
    if (e != cudaSuccess) return lv_cuda_fail(e);
    temps_.push_back(*t);
    return LV_OK;
  }
  lv_pool* pool_;
  cudaStream_t s_;
  std::vector<void*> temps_;
  std::vector<Back> backs_;
};

template <typename T>
lv_status dev_alloc(lv_pool* pool, T** ptr, size_t count) {
  void* p = nullptr;
  if (count == 0) count = 1;
  cudaError_t e = cudaMalloc(&p, count * sizeof(T));
  if (e != cudaSuccess) return lv_cuda_fail(e);
  pool->dev_allocs.push_back(p);
  *ptr = static_cast<T*>(p);
  return LV_OK;
}

// The event pair for the next launch of kind `kind`, or nullptr when timing is off.
const lv::EventPair* timing_pair(lv_pool* pool, int kind) {
  if (!pool->timing) return nullptr;
  lv::EventPair ev{};
  if (!pool->ev_free.empty()) {
    ev = pool->ev_free.back();
    pool->ev_free.pop_back();
  } else if (cudaEventCreate(&ev.start) != cudaSuccess || cudaEventCreate(&ev.end) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  pool->ev_used[kind].push_back(ev);
  return &pool->ev_used[kind].back();
}

// True when the armed fault of this kind fires now (then it disarms).
bool fault_fires(lv_pool* pool, int32_t kind) {
  if (pool->fault_kind != kind) return false;
  if (pool->fault_after > 0) {
    --pool->fault_after;
    return false;
  }
  pool->fault_kind = LV_FAULT_NONE;
  return true;
}

// At least n timing-free events, created on first use and reused.
lv_status sync_events(lv_pool* pool, size_t n) {
  while (pool->sync_events.size() < n) {
    cudaEvent_t e;
    if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) return LV_ERR_CUDA;
    pool->sync_events.push_back(e);
  }
  return LV_OK;
}

// Drops the marks of `m` once `ev` (recorded after every transfer that marked it)
// has completed; a query that finds it still running keeps them.
cudaError_t prune_marks(cudaEvent_t ev, MarkSet& m) {
  if (m.list.empty()) return cudaSuccess;
  const cudaError_t e = cudaEventQuery(ev);
  if (e == cudaErrorNotReady) return cudaSuccess;
  if (e != cudaSuccess) return e;
  m.clear();
  return cudaSuccess;
}

// The staged data movement of n validated tasks {out page, out slot, in slot, in page}
// on `s`.  The task list is read back once; its out halves are sorted by host slot and
// so are its in halves, so that consecutive slots become one copy-engine transfer
// whatever order the blocks were listed in (a session evicted suffix first sits in
// descending slots).  Then: pack the out pages into staging in slot order; copy-engine
// runs in each direction on the side streams; unpack into the in pages; joined back
// into `s`.  Every pack precedes every unpack on `s`, so a page that an incoming block
// takes is read before it is overwritten.
lv_status staged_move_inner(lv_pool* pool, const int4* tasks_dev, int64_t n, cudaStream_t s,
                            void** staging_out, bool async) {
  const lv::DevPool& d = pool->d;
  if (n <= 0) return LV_OK;
  if ((size_t)n > pool->tasks_host_cap) return LV_ERR_INVALID;
  LV_TRY(cudaMemcpyAsync(pool->tasks_host, tasks_dev, (size_t)n * sizeof(int4), cudaMemcpyDeviceToHost, s));
  LV_TRY(cudaStreamSynchronize(s));
  // split and sort, in the second and third thirds of the page-locked task buffer
  const int4* t = pool->tasks_host;
  int4* tout = pool->tasks_host + n;
  int64_t n_out = 0, n_in = 0;
  for (int64_t i = 0; i < n; ++i)
    if (t[i].x >= 0) tout[n_out++] = make_int4(t[i].x, t[i].y, -1, -1);
  int4* tin = tout + n_out;
  for (int64_t i = 0; i < n; ++i)
    if (t[i].z >= 0) tin[n_in++] = make_int4(-1, -1, t[i].z, t[i].w);
  std::stable_sort(tout, tout + n_out, [](const int4& u, const int4& v) { return u.y < v.y; });
  std::stable_sort(tin, tin + n_in, [](const int4& u, const int4& v) { return u.z < v.z; });
  if (n_out + n_in == 0) return LV_OK;      // every task was refused (errors already set)
  const size_t pb = (size_t)d.J * d.P;
  const int64_t chunk = std::max<int64_t>(1, (int64_t)((96u << 20) / pb));
  const int64_t nchunks = (std::max(n_out, n_in) + chunk - 1) / chunk;
  lv_status st = sync_events(pool, (size_t)(2 * nchunks + 3));
  if (st != LV_OK) return st;
  cudaEvent_t* ev = pool->sync_events.data();
  cudaEvent_t ev_start = ev[0];
  cudaEvent_t* ev_pack = ev + 3;            // [nchunks]
  cudaEvent_t* ev_h2d = ev + 3 + nchunks;   // [nchunks]
  // staging: out run [n_out][2L][P], in run [n_in][2L][P], then the sorted task lists, in
  // the pool's run b (alternate calls); `s` waits until the call that used run b last is
  // done with it, and the run grows (with a quarter to spare) when this call needs more
  const int b = (int)(pool->st_seq++ & 1u);
  *staging_out = &pool->st_buf[b];
  if (pool->st_buf_used[b]) LV_TRY(cudaStreamWaitEvent(s, pool->st_buf_done[b], 0));
  pool->st_buf_used[b] = true;
  {
    const size_t bytes = (size_t)(n_out + n_in) * pb + (size_t)(n_out + n_in) * sizeof(int4);
    if (bytes > pool->st_buf_bytes[b]) {
      if (pool->st_buf[b]) LV_TRY(cudaFreeAsync(pool->st_buf[b], s));
      pool->st_buf[b] = nullptr;
      pool->st_buf_bytes[b] = 0;
      const size_t want = (bytes + bytes / 4 + (64u << 20) - 1) / (64u << 20) * (64u << 20);
      cudaError_t e = cudaMallocFromPoolAsync(&pool->st_buf[b], want, pool->mp, s);
      if (e != cudaSuccess) {
        pool->st_buf[b] = nullptr;
        return lv_cuda_fail(e);
      }
      pool->st_buf_bytes[b] = want;
    }
  }
  void* staging = pool->st_buf[b];
  uint8_t* stg_out = static_cast<uint8_t*>(staging);
  uint8_t* stg_in = stg_out + (size_t)n_out * pb;
  int4* tout_dev = reinterpret_cast<int4*>(stg_in + (size_t)n_in * pb);
  int4* tin_dev = tout_dev + n_out;
  LV_TRY(cudaMemcpyAsync(tout_dev, tout, (size_t)(n_out + n_in) * sizeof(int4), cudaMemcpyHostToDevice, s));
  uint8_t* host = static_cast<uint8_t*>(pool->host_base);
  LV_TRY(cudaEventRecord(ev_start, s));
  LV_TRY(cudaStreamWaitEvent(pool->s_d2h, ev_start, 0));
  LV_TRY(cudaStreamWaitEvent(pool->s_h2d, ev_start, 0));
  if (async && pool->st_pending) {
    // Earlier asynchronous calls: a block one wrote out may come back now, a slot one
    // read may be written now, a page one loaded may be packed now.  Marks of
    // transfers that have finished are dropped; the event of a direction is waited
    // for only when this call touches a page or slot still marked for it.  Each event
    // was recorded after every earlier transfer of its stream, so one wait covers all.
    LV_TRY(prune_marks(pool->ev_st_unpack, pool->st_loaded));
    LV_TRY(prune_marks(pool->ev_st_d2h, pool->st_written));
    LV_TRY(prune_marks(pool->ev_st_h2d, pool->st_read));
    bool h2d_after_d2h = false, d2h_after_h2d = false, pack_after_unpack = false;
    for (int64_t i = 0; i < n_in && !h2d_after_d2h; ++i) h2d_after_d2h = pool->st_written.has(tin[i].z);
    for (int64_t i = 0; i < n_out && !(d2h_after_h2d && pack_after_unpack); ++i) {
      d2h_after_h2d = d2h_after_h2d || pool->st_read.has(tout[i].y);
      pack_after_unpack = pack_after_unpack || pool->st_loaded.has(tout[i].x);
    }
    if (h2d_after_d2h) LV_TRY(cudaStreamWaitEvent(pool->s_h2d, pool->ev_st_d2h, 0));
    if (d2h_after_h2d) LV_TRY(cudaStreamWaitEvent(pool->s_d2h, pool->ev_st_h2d, 0));
    if (pack_after_unpack) LV_TRY(cudaStreamWaitEvent(s, pool->ev_st_unpack, 0));
  }
  if (async) {
    for (int64_t i = 0; i < n_in; ++i) {
      pool->st_loaded.add(tin[i].w);
      pool->st_read.add(tin[i].z);
    }
    for (int64_t i = 0; i < n_out; ++i) pool->st_written.add(tout[i].y);
  }
  // H2D first so that the inbound copies start at once: runs of consecutive slots
  for (int64_t c = 0; c * chunk < n_in; ++c) {
    const int64_t a = c * chunk, b = std::min(n_in, a + chunk);
    for (int64_t i = a; i < b;) {
      int64_t j = i + 1;
      while (j < b && tin[j].z == tin[j - 1].z + 1) ++j;
      if (fault_fires(pool, LV_FAULT_COPY)) return LV_ERR_CUDA;
      LV_TRY(cudaMemcpyAsync(stg_in + (size_t)i * pb, host + (size_t)tin[i].z * pb, (size_t)(j - i) * pb,
                             cudaMemcpyHostToDevice, pool->s_h2d));
      i = j;
    }
    LV_TRY(cudaEventRecord(ev_h2d[c], pool->s_h2d));
  }
  // pack every chunk on s; the D2H runs of chunk c follow its pack
  for (int64_t c = 0; c * chunk < n_out; ++c) {
    const int64_t a = c * chunk, b = std::min(n_out, a + chunk);
    LV_TRY(lv::launch_stage(d, true, tout_dev, a, b, stg_out, s, pool->stage_ctas,
                            timing_pair(pool, LV_TIMING_PACK), pool->stage_tma));
    LV_TRY(cudaEventRecord(ev_pack[c], s));
    LV_TRY(cudaStreamWaitEvent(pool->s_d2h, ev_pack[c], 0));
    for (int64_t i = a; i < b;) {
      int64_t j = i + 1;
      while (j < b && tout[j].y == tout[j - 1].y + 1) ++j;
      if (fault_fires(pool, LV_FAULT_COPY)) return LV_ERR_CUDA;
      LV_TRY(cudaMemcpyAsync(host + (size_t)tout[i].y * pb, stg_out + (size_t)i * pb, (size_t)(j - i) * pb,
                             cudaMemcpyDeviceToHost, pool->s_d2h));
      i = j;
    }
  }
  // unpack each chunk once it has arrived, after every pack (on s, or on s_unpack
  // when asynchronous)
  cudaStream_t us = s;
  if (async) {
    us = pool->s_unpack;
    LV_TRY(cudaEventRecord(pool->ev_st_packed, s));
    LV_TRY(cudaStreamWaitEvent(us, pool->ev_st_packed, 0));
  }
  for (int64_t c = 0; c * chunk < n_in; ++c) {
    const int64_t a = c * chunk, b = std::min(n_in, a + chunk);
    LV_TRY(cudaStreamWaitEvent(us, ev_h2d[c], 0));
    LV_TRY(lv::launch_stage(d, false, tin_dev, a, b, stg_in, us, pool->stage_ctas,
                            timing_pair(pool, LV_TIMING_UNPACK), pool->stage_tma));
  }
  return LV_OK;
}

// staged_move_inner, then (also after an early error) join the side streams back
// into `s` and mark the staging run free in stream order.
lv_status staged_move(lv_pool* pool, const int4* tasks_dev, int64_t n, cudaStream_t s,
                      bool async = false) {
  void* slot = nullptr;   // &pool->st_buf[b] once the call has taken run b
  const lv_status st = staged_move_inner(pool, tasks_dev, n, s, &slot, async);
  if (!slot) return st;
  const int b = static_cast<void**>(slot) == &pool->st_buf[0] ? 0 : 1;
  if (async && st == LV_OK) {
    // the next asynchronous calls order themselves on these; run b is free again once
    // both directions and the unpacks are done
    cudaEventRecord(pool->ev_st_d2h, pool->s_d2h);
    cudaEventRecord(pool->ev_st_h2d, pool->s_h2d);
    cudaEventRecord(pool->ev_st_unpack, pool->s_unpack);
    cudaStreamWaitEvent(pool->s_unpack, pool->ev_st_d2h, 0);
    cudaStreamWaitEvent(pool->s_unpack, pool->ev_st_h2d, 0);
    cudaEventRecord(pool->st_buf_done[b], pool->s_unpack);
    cudaEventRecord(pool->ev_st_done, pool->s_unpack);
    pool->st_pending = true;
    return st;
  }
  cudaEvent_t* ev = pool->sync_events.data();
  cudaEventRecord(ev[1], pool->s_d2h);
  cudaEventRecord(ev[2], pool->s_h2d);
  cudaStreamWaitEvent(s, ev[1], 0);
  cudaStreamWaitEvent(s, ev[2], 0);
  if (async) {   // stopped early: everything joins the caller's stream
    cudaEventRecord(pool->ev_st_unpack, pool->s_unpack);
    cudaStreamWaitEvent(s, pool->ev_st_unpack, 0);
  }
  cudaEventRecord(pool->st_buf_done[b], s);
  return st;
}

// Makes `s` wait for every asynchronous page copy issued so far (with
// staged = false: not for the asynchronous staged exchanges, which order
// themselves against each other).
cudaError_t join_copies(lv_pool* pool, cudaStream_t s, bool staged = true) {
  for (int b = 0; b < 2; ++b) {
    if (!pool->copied_pending[b]) continue;
    const cudaError_t e = cudaStreamWaitEvent(s, pool->ev_copied[b], 0);
    if (e != cudaSuccess) return e;
  }
  if (staged && pool->st_pending) return cudaStreamWaitEvent(s, pool->ev_st_done, 0);
  return cudaSuccess;
}

// The scratch set of the next device-driven step, ordered on `s` after the
// copy that last used it (async); a synchronous step first joins every copy.
cudaError_t next_scratch(lv_pool* pool, cudaStream_t s, bool async, const lv::ResidentScratch** rs,
                         lv::CopyOffload* off) {
  const int b = (int)(pool->rs_seq++ & 1u);
  *rs = b ? &pool->rs_alt : &pool->rs;
  if (!async) return join_copies(pool, s);
  if (pool->st_pending) {   // an asynchronous staged exchange may still move bytes
    const cudaError_t e = cudaStreamWaitEvent(s, pool->ev_st_done, 0);
    if (e != cudaSuccess) return e;
  }
  if (pool->copied_pending[b]) {
    const cudaError_t e = cudaStreamWaitEvent(s, pool->ev_copied[b], 0);
    if (e != cudaSuccess) return e;
  }
  *off = lv::CopyOffload{pool->s_copy, pool->ev_planned, pool->ev_copied[b], pool->ev_copy_start,
                         pool->ev_copy_end};
  pool->copied_pending[b] = true;
  return cudaSuccess;
}

void free_pool(lv_pool* pool) {
  for (auto& g : pool->step_graphs) {
    if (g.exec) cudaGraphExecDestroy(g.exec);
    if (g.graph) cudaGraphDestroy(g.graph);
  }
  pool->step_graphs.clear();
  if (pool->s_capture) cudaStreamDestroy(pool->s_capture);
  if (pool->s_unpack) cudaStreamSynchronize(pool->s_unpack);
  if (pool->s_unpack) cudaStreamDestroy(pool->s_unpack);
  for (cudaEvent_t e : {pool->ev_st_d2h, pool->ev_st_h2d, pool->ev_st_unpack, pool->ev_st_packed,
                        pool->ev_st_done, pool->st_buf_done[0], pool->st_buf_done[1]})
    if (e) cudaEventDestroy(e);
  if (pool->s_copy) cudaStreamSynchronize(pool->s_copy);
  if (pool->s_copy) cudaStreamDestroy(pool->s_copy);
  if (pool->ev_planned) cudaEventDestroy(pool->ev_planned);
  if (pool->ev_copy_start) cudaEventDestroy(pool->ev_copy_start);
  if (pool->ev_copy_end) cudaEventDestroy(pool->ev_copy_end);
  for (cudaEvent_t e : pool->ev_copied)
    if (e) cudaEventDestroy(e);
  for (cudaEvent_t e : pool->sync_events) cudaEventDestroy(e);
  if (pool->s_d2h) cudaStreamDestroy(pool->s_d2h);
  if (pool->s_h2d) cudaStreamDestroy(pool->s_h2d);
  if (pool->tasks_host) cudaFreeHost(pool->tasks_host);
  for (auto& v : pool->ev_used)
    for (auto& e : v) pool->ev_free.push_back(e);
  for (auto& e : pool->ev_free) {
    cudaEventDestroy(e.start);
    cudaEventDestroy(e.end);
  }
  for (void* b : pool->st_buf)
    if (b) cudaFree(b);   // after every stream above has been synchronised
  for (void* p : pool->dev_allocs) cudaFree(p);
  pool->dev_allocs.clear();
  if (pool->own_host && pool->host_base) cudaFreeHost(pool->host_base);
  if (pool->mp) cudaMemPoolDestroy(pool->mp);
  delete pool;
}

inline cudaStream_t as_stream(lv_stream s) { return static_cast<cudaStream_t>(s); }

lv_status validate_desc(const lv_pool_desc* d) {
  if (!d) return LV_ERR_INVALID;
  if (d->num_layers < 1 || d->num_kv_heads < 1 || d->head_dim < 1 || d->page_tokens < 1 ||
      d->elem_bytes < 1)
    return LV_ERR_INVALID;
  const long long P = (long long)d->page_tokens * d->num_kv_heads * d->head_dim * d->elem_bytes;
  if (P % 16 != 0 || P > (1ll << 30)) return LV_ERR_INVALID;
  if (d->num_layers > 4096) return LV_ERR_INVALID;
  if (d->max_sessions < 1 || d->max_sessions > 4096) return LV_ERR_INVALID;
  if (d->max_blocks < 1 || d->max_blocks > 65536) return LV_ERR_INVALID;
  if (d->hbm_pages < 1 || d->hbm_pages > 0x7fffffffll) return LV_ERR_INVALID;
  if (d->hbm_budget_pages < 1 || d->hbm_budget_pages > d->hbm_pages) return LV_ERR_INVALID;
  if (d->host_pages < 0 || d->host_pages > 0x7ffffffdll) return LV_ERR_INVALID;
  if (d->reply_prior_us < 0 || d->protect_us < 0) return LV_ERR_INVALID;
  if (d->unit_us < 1 || d->unit_us > (1ll << 31)) return LV_ERR_INVALID;
  if (d->t_play_mode != LV_PLAY_PLAYBACK && d->t_play_mode != LV_PLAY_COUNTERS) return LV_ERR_INVALID;
  if (d->within_order != LV_SUFFIX_FIRST && d->within_order != LV_ASCENDING) return LV_ERR_INVALID;
  if (d->policy != LV_POLICY_NEXT_USE && d->policy != LV_POLICY_LRU) return LV_ERR_INVALID;
  if (d->tiers != LV_TIERS_EXCLUSIVE && d->tiers != LV_TIERS_INCLUSIVE) return LV_ERR_INVALID;
  if (d->reserved != 0) return LV_ERR_INVALID;
  if (d->hbm_kv == nullptr) return LV_ERR_INVALID;
  return LV_OK;
}

lv_status create_impl(const lv_pool_desc* desc, cudaStream_t s, lv_pool** out) {
  lv_status st = validate_desc(desc);
  if (st != LV_OK) return st;
  lv_pool* pool = new (std::nothrow) lv_pool();
  if (!pool) return LV_ERR_OOM;
  auto fail = [&](lv_status code) {
    free_pool(pool);
    return code;
  };
  DevPool& d = pool->d;
  if (cudaGetDevice(&pool->device) != cudaSuccess) return fail(LV_ERR_CUDA);
  if (cudaDeviceGetAttribute(&pool->num_sms, cudaDevAttrMultiProcessorCount, pool->device) != cudaSuccess)
    return fail(LV_ERR_CUDA);
  d.S = desc->max_sessions;
  d.maxB = desc->max_blocks;
  d.T = desc->page_tokens;
  d.J = 2 * desc->num_layers;
  d.P = (int64_t)desc->page_tokens * desc->num_kv_heads * desc->head_dim * desc->elem_bytes;
  d.hbm_pages = desc->hbm_pages;
  d.budget = desc->hbm_budget_pages;
  d.host_pages = desc->host_pages;
  d.reply_prior_us = desc->reply_prior_us;
  d.protect_us = desc->protect_us;
  d.unit_us = desc->unit_us;
  d.within = desc->within_order;
  d.tplay = desc->t_play_mode;
  d.policy = desc->policy;
  d.incl = desc->tiers == LV_TIERS_INCLUSIVE ? 1 : 0;

  // the caller's HBM sub-page arrays
  std::vector<uint8_t*> kv(d.J);
  for (int j = 0; j < d.J; ++j) {
    void* p = desc->hbm_kv[j];
    if (!p || (reinterpret_cast<uintptr_t>(p) & 15) || !is_device_ptr(p)) return fail(LV_ERR_INVALID);
    kv[j] = static_cast<uint8_t*>(p);
  }
  // the host pool
  const size_t host_bytes = (size_t)d.host_pages * d.J * d.P;
  if (desc->host_kv) {
    cudaPointerAttributes a{};
    if (cudaPointerGetAttributes(&a, desc->host_kv) != cudaSuccess) {
      cudaGetLastError();
      return fail(LV_ERR_INVALID);
    }
    if (a.type != cudaMemoryTypeHost || a.devicePointer == nullptr ||
        (reinterpret_cast<uintptr_t>(a.devicePointer) & 15))
      return fail(LV_ERR_INVALID);
    pool->host_base = desc->host_kv;
    d.host = static_cast<uint8_t*>(a.devicePointer);
  } else if (host_bytes > 0) {
    void* h = nullptr;
    cudaError_t e = cudaHostAlloc(&h, host_bytes, cudaHostAllocMapped | cudaHostAllocPortable);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return fail(LV_ERR_OOM);
    }
    pool->own_host = true;
    pool->host_base = h;
    void* hd = nullptr;
    if (cudaHostGetDevicePointer(&hd, h, 0) != cudaSuccess) return fail(LV_ERR_CUDA);
    d.host = static_cast<uint8_t*>(hd);
  }

  uint8_t** kv_dev = nullptr;
  const size_t tb = (size_t)d.S * d.maxB;
  const size_t wh = (size_t)((d.hbm_pages + 31) / 32), wo = (size_t)((d.host_pages + 31) / 32);
  if ((st = dev_alloc(pool, &kv_dev, d.J)) != LV_OK ||
      (st = dev_alloc(pool, &d.sess, d.S)) != LV_OK ||
      (st = dev_alloc(pool, &d.table, tb)) != LV_OK ||
      (st = dev_alloc(pool, &d.mark, tb)) != LV_OK ||
      (st = dev_alloc(pool, &d.shadow, tb)) != LV_OK ||
      (st = dev_alloc(pool, &d.own_hbm, (size_t)d.hbm_pages)) != LV_OK ||
      (st = dev_alloc(pool, &d.own_host, (size_t)d.host_pages)) != LV_OK ||
      (st = dev_alloc(pool, &d.bits_hbm, wh)) != LV_OK ||
      (st = dev_alloc(pool, &d.bits_host, wo)) != LV_OK ||
      (st = dev_alloc(pool, &d.ctl, (size_t)lv::C_N)) != LV_OK ||
      (st = dev_alloc(pool, &d.skey, d.S)) != LV_OK ||
      (st = dev_alloc(pool, &d.scount, d.S)) != LV_OK ||
      (st = dev_alloc(pool, &d.sbefore, d.S)) != LV_OK ||
      (st = dev_alloc(pool, &d.page_tag, (size_t)d.hbm_pages)) != LV_OK)
    return fail(st);
  lv::ResidentScratch& rs = pool->rs;
  if ((st = dev_alloc(pool, &rs.victims, (size_t)d.budget)) != LV_OK ||
      (st = dev_alloc(pool, &rs.slots, (size_t)d.budget)) != LV_OK ||
      (st = dev_alloc(pool, &rs.blocks, (size_t)d.maxB)) != LV_OK ||
      (st = dev_alloc(pool, &rs.loads, (size_t)d.maxB)) != LV_OK ||
      (st = dev_alloc(pool, &rs.pages, (size_t)d.maxB)) != LV_OK ||
      (st = dev_alloc(pool, &rs.append, (size_t)d.maxB + 2)) != LV_OK ||
      (st = dev_alloc(pool, &rs.tasks, (size_t)d.budget + d.maxB)) != LV_OK ||
      (st = dev_alloc(pool, &rs.words, 16)) != LV_OK ||
      (st = dev_alloc(pool, &rs.hits, (size_t)d.S)) != LV_OK ||
      (st = dev_alloc(pool, &pool->sched_scratch, (size_t)32 * LV_SCHED_MAX_REQUESTS)) != LV_OK)
    return fail(st);
  pool->rs_alt = rs;
  if ((st = dev_alloc(pool, &pool->rs_alt.tasks, (size_t)d.budget + d.maxB)) != LV_OK ||
      (st = dev_alloc(pool, &pool->rs_alt.words, 16)) != LV_OK)
    return fail(st);
  // asynchronous turn copies gate the turn's start: their CTAs are scheduled first
  int prio_least = 0, prio_greatest = 0;
  if (cudaDeviceGetStreamPriorityRange(&prio_least, &prio_greatest) != cudaSuccess) prio_greatest = 0;
  if (cudaStreamCreateWithPriority(&pool->s_copy, cudaStreamNonBlocking, prio_greatest) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->ev_planned, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->ev_copy_start, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->ev_copy_end, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->ev_copied[0], cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->ev_copied[1], cudaEventDisableTiming) != cudaSuccess)
    return fail(LV_ERR_CUDA);
  d.kv = kv_dev;
  if (cudaMemcpyAsync(kv_dev, kv.data(), d.J * sizeof(uint8_t*), cudaMemcpyHostToDevice, s) != cudaSuccess ||
      cudaMemsetAsync(d.sess, 0, d.S * sizeof(lv_session_state), s) != cudaSuccess ||
      cudaMemsetAsync(d.table, 0xff, tb * sizeof(int32_t), s) != cudaSuccess ||
      cudaMemsetAsync(d.mark, 0, tb * sizeof(int32_t), s) != cudaSuccess ||
      cudaMemsetAsync(d.shadow, 0xff, tb * sizeof(int32_t), s) != cudaSuccess ||
      cudaMemsetAsync(d.own_hbm, 0xff, (size_t)d.hbm_pages * 4, s) != cudaSuccess ||
      cudaMemsetAsync(d.own_host, 0xff, (size_t)(d.host_pages ? d.host_pages : 1) * 4, s) != cudaSuccess ||
      cudaMemsetAsync(d.bits_hbm, 0, wh * 4, s) != cudaSuccess ||
      cudaMemsetAsync(d.bits_host, 0, (wo ? wo : 1) * 4, s) != cudaSuccess ||
      cudaMemsetAsync(d.ctl, 0, lv::C_N * sizeof(long long), s) != cudaSuccess ||
      cudaMemsetAsync(d.page_tag, 0, (size_t)d.hbm_pages * 8, s) != cudaSuccess)
    return fail(LV_ERR_CUDA);
  // A fifth of the SMs (30 CTAs on GB300) keeps both link directions saturated (338 GB/s,
  // the same as 50 CTAs or one per SM; 25 CTAs fall to 326) and leaves the rest of the
  // GPU to the serving work that runs meanwhile: next to a consumer reading resident KV
  // at HBM speed, 30 CTAs moved 211 GB/s and left it 0.88 of its rate, against 197 GB/s
  // and 0.835 for 50 CTAs and 167 GB/s and 0.67 for 152.
  // 3/10 of the SMs (45 on GB300): the fewest CTAs that keep both link directions busy
  // alone, and most of the link next to a kernel that reads HBM on every SM
  pool->exchange_ctas = pool->num_sms * 3 / 10 > 0 ? pool->num_sms * 3 / 10 : 1;
  if (const char* env = std::getenv("LV_EXCHANGE_CTAS_PER_SM")) {
    const int per = std::atoi(env);
    if (per >= 1 && per <= 16) pool->exchange_ctas = pool->num_sms * per;
  }
  if (const char* env = std::getenv("LV_EXCHANGE_CTAS")) {   // an explicit grid (1 .. 16 per SM)
    const int n = std::atoi(env);
    if (n >= 1 && n <= pool->num_sms * 16) pool->exchange_ctas = n;
  }

  // the exchange copy: 16-byte SM loads and stores by default; LV_EXCHANGE_KERNEL=tma
  // moves it with TMA bulk copies through LV_EXCHANGE_STAGES (default 4) stages of 2P
  // bytes per CTA, where two stages fit in a CTA's shared memory
  d.xstages = 0;
  if (const char* env = std::getenv("LV_EXCHANGE_KERNEL")) {
    if (std::strcmp(env, "tma") == 0) {
      int st = 4;
      if (const char* e2 = std::getenv("LV_EXCHANGE_STAGES")) st = std::atoi(e2);
      const int lim = lv::exchange_stage_limit(d.P);
      if (st > lim) st = lim;
      d.xstages = st >= 2 ? st : 0;
    }
  }
  if (lv::configure_exchange_tma(d) != cudaSuccess) return fail(LV_ERR_CUDA);
  if (const char* env = std::getenv("LV_STAGE_STAGES")) {   // TMA pack/unpack stages per CTA
    const int st = std::atoi(env);
    if (st >= 2 && st <= 16) d.stages = st;
  }
  // two TMA stages must fit in a CTA's shared memory; larger sub-pages use 16-byte copies
  const bool tma_fits = 2 * d.P <= 227 * 1024;
  if (tma_fits && lv::configure_stage_kernels(d) != cudaSuccess) return fail(LV_ERR_CUDA);
  if (cudaStreamCreateWithFlags(&pool->s_d2h, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&pool->s_h2d, cudaStreamNonBlocking) != cudaSuccess ||
      cudaStreamCreateWithFlags(&pool->s_unpack, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->ev_st_d2h, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->ev_st_h2d, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->ev_st_unpack, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->ev_st_packed, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->ev_st_done, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->st_buf_done[0], cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&pool->st_buf_done[1], cudaEventDisableTiming) != cudaSuccess)
    return fail(LV_ERR_CUDA);
  pool->tasks_host_cap = (size_t)d.budget + d.maxB + (size_t)d.host_pages;
  pool->st_loaded.resize(d.hbm_pages);
  pool->st_written.resize(d.host_pages);
  pool->st_read.resize(d.host_pages);
  // the task list read back, then its sorted out and in halves
  if (cudaHostAlloc((void**)&pool->tasks_host, 3 * pool->tasks_host_cap * sizeof(int4), cudaHostAllocDefault) !=
      cudaSuccess) {
    pool->tasks_host = nullptr;
    return fail(LV_ERR_OOM);
  }
  pool->stage_ctas = 2 * pool->num_sms;   // two TMA pack/unpack CTAs per SM (see stage_count)
  if (const char* env = std::getenv("LV_STAGE_CTAS_PER_SM")) {
    const int per = std::atoi(env);
    if (per >= 1 && per <= 4) pool->stage_ctas = pool->num_sms * per;
  }
  if (const char* env = std::getenv("LV_STAGE_KERNEL")) pool->stage_tma = std::strcmp(env, "lsu") != 0;
  // device-driven steps on the caller's stream as graph launches (LV_STEP_GRAPHS=0: one
  // kernel launch at a time)
  if (const char* env = std::getenv("LV_STEP_GRAPHS")) pool->step_graphs_on = std::strcmp(env, "0") != 0;
  if (const char* env = std::getenv("LV_REMAP_ENTRIES_PER_THREAD")) {   // 1, 2 or 4
    const int e = std::atoi(env);
    if (e == 1 || e == 2 || e == 4) pool->remap_per_thread = e;
  }
  if (!tma_fits) pool->stage_tma = false;
  cudaMemPoolProps props{};
  props.allocType = cudaMemAllocationTypePinned;
  props.location.type = cudaMemLocationTypeDevice;
  props.location.id = pool->device;
  if (cudaMemPoolCreate(&pool->mp, &props) != cudaSuccess) {
    pool->mp = nullptr;
    return fail(LV_ERR_CUDA);
  }
  uint64_t threshold = UINT64_MAX;
  cudaMemPoolSetAttribute(pool->mp, cudaMemPoolAttrReleaseThreshold, &threshold);
  // never make one stream wait for another to reuse a freed run (asynchronous staged
  // exchanges free on their own stream): grow the pool instead
  int no_internal = 0;
  cudaMemPoolSetAttribute(pool->mp, cudaMemPoolReuseAllowInternalDependencies, &no_internal);
  if (cudaStreamSynchronize(s) != cudaSuccess) return fail(LV_ERR_CUDA);
  *out = pool;
  return LV_OK;
}

// The kernel nodes of a captured launch chain, in launch order (each node depends on
// the one before it); false unless the graph is exactly such a chain of n nodes.
bool chain_nodes(cudaGraph_t graph, size_t n, std::vector<cudaGraphNode_t>* order) {
  size_t count = 0;
  if (cudaGraphGetNodes(graph, nullptr, &count) != cudaSuccess || count != n) return false;
  std::vector<cudaGraphNode_t> nodes(count);
  if (cudaGraphGetNodes(graph, nodes.data(), &count) != cudaSuccess) return false;
  std::vector<cudaGraphNode_t> prev(count, nullptr);
  cudaGraphNode_t root = nullptr;
  for (size_t i = 0; i < count; ++i) {
    // with room for two, so that a node with more than one dependency is seen; the edge
    // data is asked for too (programmatic edges are not default edges)
    cudaGraphNode_t deps[2] = {nullptr, nullptr};
    cudaGraphEdgeData edge[2] = {};
    size_t nd = 2;
    if (cudaGraphNodeGetDependencies(nodes[i], deps, edge, &nd) != cudaSuccess || nd > 1) return false;
    if (nd == 1) {
      prev[i] = deps[0];
    } else if (root) {
      return false;
    } else {
      root = nodes[i];
    }
  }
  order->clear();
  for (cudaGraphNode_t cur = root; cur && order->size() < count;) {
    order->push_back(cur);
    cudaGraphNode_t next = nullptr;
    for (size_t i = 0; i < count; ++i)
      if (prev[i] == cur) next = nodes[i];
    cur = next;
  }
  for (cudaGraphNode_t nd : *order) {
    cudaGraphNodeType t;
    if (cudaGraphNodeGetType(nd, &t) != cudaSuccess || t != cudaGraphNodeTypeKernel) return false;
  }
  return order->size() == count;
}

// Issues a device-driven step whose kernels all run on `s` (`launch(stream)` makes its
// launches): the launches are recorded, and the instantiated graph of the same shape
// (built by stream capture on first use) is launched with every kernel node's arguments
// replaced by this step's.  A shape that cannot be captured as a chain turns the graphs
// off for the pool, and the recorded launches are issued one by one.
template <typename F>
cudaError_t run_step(lv_pool* pool, cudaStream_t s, F&& launch) {
  if (!pool->step_graphs_on) return launch(s);
  std::vector<lv::LaunchRecord> recs;
  lv::set_launch_recorder(&recs);
  cudaError_t e = launch(s);
  lv::set_launch_recorder(nullptr);
  if (e != cudaSuccess || recs.empty()) return e;
  lv_pool::StepGraph* g = nullptr;
  for (auto& c : pool->step_graphs) {
    if (c.funcs.size() != recs.size()) continue;
    bool same = true;
    for (size_t i = 0; i < recs.size() && same; ++i)
      same = c.funcs[i] == recs[i].func && c.grids[i].x == recs[i].grid.x && c.grids[i].y == recs[i].grid.y &&
             c.blocks[i].x == recs[i].block.x && c.smems[i] == recs[i].smem;
    if (same) {
      g = &c;
      break;
    }
  }
  if (g) {
    for (size_t i = 0; i < recs.size(); ++i) {
      cudaKernelNodeParams kp{};
      kp.func = const_cast<void*>(recs[i].func);
      kp.gridDim = recs[i].grid;
      kp.blockDim = recs[i].block;
      kp.sharedMemBytes = (unsigned)recs[i].smem;
      kp.kernelParams = const_cast<void**>(recs[i].args.data());
      e = cudaGraphExecKernelNodeSetParams(g->exec, g->nodes[i], &kp);
      if (e != cudaSuccess) return e;
    }
    return cudaGraphLaunch(g->exec, s);
  }
  // a new shape: capture the launches on the pool's capture stream (past 32 shapes,
  // further shapes are issued launch by launch)
  if (pool->step_graphs.size() >= 32) return lv::replay_launches(recs, s);
  lv_pool::StepGraph c;
  bool ok = true;
  if (!pool->s_capture) ok = cudaStreamCreateWithFlags(&pool->s_capture, cudaStreamNonBlocking) == cudaSuccess;
  if (ok) ok = cudaStreamBeginCapture(pool->s_capture, cudaStreamCaptureModeThreadLocal) == cudaSuccess;
  if (ok) {
    const cudaError_t le = lv::replay_launches(recs, pool->s_capture);
    const cudaError_t ce = cudaStreamEndCapture(pool->s_capture, &c.graph);
    ok = le == cudaSuccess && ce == cudaSuccess && c.graph;
  }
  if (ok) ok = chain_nodes(c.graph, recs.size(), &c.nodes);
  if (ok) ok = cudaGraphInstantiate(&c.exec, c.graph, 0) == cudaSuccess;
  if (!ok) {
    cudaGetLastError();
    if (c.exec) cudaGraphExecDestroy(c.exec);
    if (c.graph) cudaGraphDestroy(c.graph);
    pool->step_graphs_on = false;
    return lv::replay_launches(recs, s);
  }
  for (const auto& r : recs) {
    c.funcs.push_back(r.func);
    c.grids.push_back(r.grid);
    c.blocks.push_back(r.block);
    c.smems.push_back(r.smem);
  }
  pool->step_graphs.push_back(std::move(c));
  return cudaGraphLaunch(pool->step_graphs.back().exec, s);
}

}  // namespace

namespace lv {
void pool_shape(const lv_pool* pool, int32_t* sessions, int32_t* max_blocks, int64_t* page_bytes,
                int64_t* budget, int64_t* host_pages) {
  *sessions = pool->d.S;
  *max_blocks = pool->d.maxB;
  *page_bytes = (int64_t)pool->d.J * pool->d.P;
  *budget = pool->d.budget;
  *host_pages = pool->d.host_pages;
}
}  // namespace lv

extern "C" {

lv_status lv_pool_create(const lv_pool_desc* desc, lv_stream stream, lv_pool** out) {
  NvtxRange nvtx_range("lv_pool_create");
  if (!out) return LV_ERR_INVALID;
  *out = nullptr;
  try {
    return create_impl(desc, as_stream(stream), out);
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_pool_destroy(lv_pool* pool, lv_stream stream) {
  NvtxRange nvtx_range("lv_pool_destroy");
  if (!pool) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  cudaError_t e = join_copies(pool, as_stream(stream));
  if (e == cudaSuccess) e = cudaStreamSynchronize(as_stream(stream));
  free_pool(pool);
  return e == cudaSuccess ? LV_OK : LV_ERR_CUDA;
}

void* lv_pool_host_ptr(lv_pool* pool) { return pool ? pool->host_base : nullptr; }

lv_status lv_pool_import(lv_pool* pool, const int32_t* placement, const int32_t* ctx_tokens,
                         lv_stream stream) {
  NvtxRange nvtx_range("lv_pool_import");
  if (!pool || !placement || !ctx_tokens) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  DevPool& d = pool->d;
  try {
    LV_TRY(join_copies(pool, s));   // a new placement: no copy of the old one may still run
    Staging st(pool, s);
    const void *pl = nullptr, *cx = nullptr;
    lv_status r;
    if ((r = st.in(placement, (size_t)d.S * d.maxB * 4, &pl)) != LV_OK) return r;
    if ((r = st.in(ctx_tokens, (size_t)d.S * 4, &cx)) != LV_OK) return r;
    LV_TRY(cudaMemsetAsync(d.own_hbm, 0xff, (size_t)d.hbm_pages * 4, s));
    if (d.host_pages) LV_TRY(cudaMemsetAsync(d.own_host, 0xff, (size_t)d.host_pages * 4, s));
    LV_TRY(cudaMemsetAsync(d.bits_hbm, 0, (size_t)((d.hbm_pages + 31) / 32) * 4, s));
    if (d.host_pages) LV_TRY(cudaMemsetAsync(d.bits_host, 0, (size_t)((d.host_pages + 31) / 32) * 4, s));
    LV_TRY(cudaMemsetAsync(d.ctl, 0, 2 * sizeof(long long), s));   // allocation counts
    LV_TRY(cudaMemsetAsync(d.ctl + lv::C_CLEAN, 0, sizeof(long long), s));   // no clean copies
    LV_TRY(lv::launch_import(d, static_cast<const int32_t*>(pl), static_cast<const int32_t*>(cx), s));
    LV_TRY(lv::launch_check_budget(d, s));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_session_set(lv_pool* pool, const lv_session_state* states, int32_t first, int32_t n,
                         lv_stream stream) {
  NvtxRange nvtx_range("lv_session_set");
  if (!pool || first < 0 || n < 0 || (long long)first + n > pool->d.S) return LV_ERR_INVALID;
  if (n == 0) return LV_OK;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    Staging st(pool, s);
    const void* in = nullptr;
    lv_status r = st.in(states, (size_t)n * sizeof(lv_session_state), &in);
    if (r != LV_OK) return r;
    LV_TRY(lv::launch_session_set(pool->d, static_cast<const lv_session_state*>(in), first, n, s));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_session_get(lv_pool* pool, lv_session_state* out, int32_t first, int32_t n,
                         lv_stream stream) {
  if (!pool || !out || first < 0 || n < 0 || (long long)first + n > pool->d.S) return LV_ERR_INVALID;
  if (n == 0) return LV_OK;
  DeviceGuard g(pool->device);
  LV_TRY(cudaMemcpyAsync(out, pool->d.sess + first, (size_t)n * sizeof(lv_session_state),
                         cudaMemcpyDefault, as_stream(stream)));
  return LV_OK;
}

lv_status lv_session_events(lv_pool* pool, const lv_event* events, int64_t n, lv_stream stream) {
  NvtxRange nvtx_range("lv_session_events");
  if (!pool || n < 0 || (n > 0 && !events)) return LV_ERR_INVALID;
  if (n == 0) return LV_OK;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    Staging st(pool, s);
    const void* in = nullptr;
    lv_status r = st.in(events, (size_t)n * sizeof(lv_event), &in);
    if (r != LV_OK) return r;
    LV_TRY(lv::launch_events(pool->d, static_cast<const lv_event*>(in), n, s));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_select_victims(lv_pool* pool, int64_t now_us, int64_t k, uint32_t flags,
                            lv_victim* out, int64_t capacity, int64_t* count_out,
                            lv_stream stream) {
  NvtxRange nvtx_range("lv_select_victims");
  if (!pool || k < 0 || capacity < 0 || (flags & ~(uint32_t)LV_SELECT_FALLBACK)) return LV_ERR_INVALID;
  const int64_t keff = k < capacity ? k : capacity;
  if (keff > 0 && !out) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    Staging st(pool, s);
    void *vdev = nullptr, *cdev = nullptr;
    lv_status r;
    if ((r = st.out(out, (size_t)keff * sizeof(lv_victim), &vdev, false)) != LV_OK) return r;
    if ((r = st.out(count_out, sizeof(int64_t), &cdev, false)) != LV_OK) return r;
    LV_TRY(lv::launch_select(pool->d, now_us, keff, (flags & LV_SELECT_FALLBACK) != 0,
                             static_cast<lv_victim*>(vdev), static_cast<long long*>(cdev), s,
                             pool->num_sms));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_swap_out(lv_pool* pool, const lv_victim* victims, int64_t n, int32_t* slots_out,
                      lv_remap_entry* commit_out, int32_t mode, lv_stream stream) {
  NvtxRange nvtx_range("lv_swap_out");
  if (!pool || n < 0 || n > 0x7fffffffll || (n > 0 && !victims)) return LV_ERR_INVALID;
  if (mode != LV_MODE_AUTO && mode != LV_MODE_ZERO_COPY && mode != LV_MODE_STAGED) return LV_ERR_INVALID;
  if (n == 0) return LV_OK;
  if (pool->d.host_pages == 0) return LV_ERR_INVALID;
  if (mode == LV_MODE_STAGED && (size_t)n > pool->tasks_host_cap) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    LV_TRY(join_copies(pool, s));   // earlier asynchronous copies move bytes too
    Staging st(pool, s);
    const void* vin = nullptr;
    void *sdev = nullptr, *cdev = nullptr;
    lv_status r;
    if ((r = st.in(victims, (size_t)n * sizeof(lv_victim), &vin)) != LV_OK) return r;
    if ((r = st.out(slots_out, (size_t)n * 4, &sdev, true)) != LV_OK) return r;
    if ((r = st.out(commit_out, (size_t)n * sizeof(lv_remap_entry), &cdev, false)) != LV_OK) return r;
    int32_t* slots = static_cast<int32_t*>(sdev);
    const bool fail_alloc = fault_fires(pool, LV_FAULT_HOST_ALLOC);
    if (pool->d.incl)
      LV_TRY(lv::launch_alloc_out(pool->d, static_cast<const lv_victim*>(vin), n, slots, s, fail_alloc));
    else
      LV_TRY(lv::launch_alloc(pool->d, false, n, slots, s, fail_alloc));
    if (mode == LV_MODE_STAGED) {
      void* tdev = nullptr;
      if ((r = st.out(nullptr, (size_t)n * sizeof(int4), &tdev, true)) != LV_OK) return r;
      LV_TRY(lv::launch_tasks_out(pool->d, static_cast<const lv_victim*>(vin), slots, n,
                                  static_cast<int4*>(tdev), static_cast<lv_remap_entry*>(cdev), s));
      if ((r = staged_move(pool, static_cast<int4*>(tdev), n, s)) != LV_OK) return r;
      return st.finish();
    }
    LV_TRY(lv::launch_swap_out(pool->d, static_cast<const lv_victim*>(vin), slots, n,
                               static_cast<lv_remap_entry*>(cdev), s, pool->num_sms,
                               timing_pair(pool, LV_TIMING_SWAP_OUT)));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_swap_in(lv_pool* pool, int32_t sid, const int32_t* blks, int64_t n, int32_t* pages_out,
                     lv_remap_entry* commit_out, int32_t mode, lv_stream stream) {
  NvtxRange nvtx_range("lv_swap_in");
  if (!pool || n < 0 || n > 0x7fffffffll || (n > 0 && !blks)) return LV_ERR_INVALID;
  if (mode != LV_MODE_AUTO && mode != LV_MODE_ZERO_COPY && mode != LV_MODE_STAGED) return LV_ERR_INVALID;
  if (sid < 0 || sid >= pool->d.S) return LV_ERR_INVALID;
  if (mode == LV_MODE_STAGED && (size_t)n > pool->tasks_host_cap) return LV_ERR_INVALID;
  if (n == 0) return LV_OK;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    LV_TRY(join_copies(pool, s));   // earlier asynchronous copies move bytes too
    Staging st(pool, s);
    const void* bin = nullptr;
    void *pdev = nullptr, *cdev = nullptr;
    lv_status r;
    if ((r = st.in(blks, (size_t)n * 4, &bin)) != LV_OK) return r;
    if ((r = st.out(pages_out, (size_t)n * 4, &pdev, true)) != LV_OK) return r;
    if ((r = st.out(commit_out, (size_t)n * sizeof(lv_remap_entry), &cdev, false)) != LV_OK) return r;
    int32_t* pages = static_cast<int32_t*>(pdev);
    LV_TRY(lv::launch_alloc(pool->d, true, n, pages, s, fault_fires(pool, LV_FAULT_HBM_ALLOC)));
    if (mode == LV_MODE_STAGED) {
      void* tdev = nullptr;
      if ((r = st.out(nullptr, (size_t)n * sizeof(int4), &tdev, true)) != LV_OK) return r;
      LV_TRY(lv::launch_tasks_in(pool->d, sid, static_cast<const int32_t*>(bin), pages, n,
                                 static_cast<int4*>(tdev), static_cast<lv_remap_entry*>(cdev), s));
      if ((r = staged_move(pool, static_cast<int4*>(tdev), n, s)) != LV_OK) return r;
      return st.finish();
    }
    LV_TRY(lv::launch_swap_in(pool->d, sid, static_cast<const int32_t*>(bin), pages, n,
                              static_cast<lv_remap_entry*>(cdev), s, pool->num_sms,
                              timing_pair(pool, LV_TIMING_SWAP_IN)));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_swap_exchange(lv_pool* pool, const lv_victim* victims, int64_t n_out, int32_t sid,
                           const int32_t* blks, int64_t n_in, int32_t* slots_out, int32_t* pages_out,
                           int32_t mode, lv_stream stream) {
  NvtxRange nvtx_range("lv_swap_exchange");
  if (!pool || n_out < 0 || n_in < 0 || n_out > 0x7fffffffll || n_in > 0x7fffffffll ||
      (n_out > 0 && !victims) || (n_in > 0 && !blks))
    return LV_ERR_INVALID;
  const bool async = (mode & LV_MODE_ASYNC) != 0;
  mode &= ~LV_MODE_ASYNC;
  if (mode != LV_MODE_AUTO && mode != LV_MODE_ZERO_COPY && mode != LV_MODE_STAGED) return LV_ERR_INVALID;
  if (async && mode != LV_MODE_STAGED) return LV_ERR_INVALID;
  if (n_in > 0 && (sid < 0 || sid >= pool->d.S)) return LV_ERR_INVALID;
  if (mode == LV_MODE_STAGED && (size_t)(n_out + n_in) > pool->tasks_host_cap) return LV_ERR_INVALID;
  if (n_out > 0 && pool->d.host_pages == 0) return LV_ERR_INVALID;
  if (n_out == 0 && n_in == 0) return LV_OK;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    // earlier asynchronous copies move bytes too (an asynchronous staged exchange
    // orders itself against the previous one, transfer by transfer)
    LV_TRY(join_copies(pool, s, !async));
    Staging st(pool, s);
    const void *vin = nullptr, *bin = nullptr;
    void *sdev = nullptr, *pdev = nullptr, *tdev = nullptr, *ndev = nullptr;
    lv_status r;
    if ((r = st.in(victims, (size_t)n_out * sizeof(lv_victim), &vin)) != LV_OK) return r;
    if ((r = st.in(blks, (size_t)n_in * 4, &bin)) != LV_OK) return r;
    if ((r = st.out(slots_out, (size_t)n_out * 4, &sdev, true)) != LV_OK) return r;
    if ((r = st.out(pages_out, (size_t)n_in * 4, &pdev, true)) != LV_OK) return r;
    if ((r = st.out(nullptr, (size_t)(n_out + n_in) * sizeof(int4), &tdev, true)) != LV_OK) return r;
    // the task count, and the copy kernel's cursor
    if ((r = st.out(nullptr, 2 * sizeof(long long), &ndev, true)) != LV_OK) return r;
    if (++pool->epoch <= 0) pool->epoch = 1;
    if (mode == LV_MODE_STAGED) {
      LV_TRY(lv::launch_exchange_plan(pool->d, static_cast<const lv_victim*>(vin), n_out, sid,
                                      static_cast<const int32_t*>(bin), n_in, static_cast<int32_t*>(sdev),
                                      static_cast<int32_t*>(pdev), static_cast<int4*>(tdev),
                                      static_cast<long long*>(ndev), pool->epoch, pool->d.page_tag, s));
      long long nt = 0;
      LV_TRY(cudaMemcpyAsync(&nt, ndev, sizeof(nt), cudaMemcpyDeviceToHost, s));
      LV_TRY(cudaStreamSynchronize(s));
      if ((r = staged_move(pool, static_cast<int4*>(tdev), nt, s, async)) != LV_OK) return r;
      return st.finish();
    }
    LV_TRY(lv::launch_exchange(pool->d, static_cast<const lv_victim*>(vin), n_out, sid,
                               static_cast<const int32_t*>(bin), n_in, static_cast<int32_t*>(sdev),
                               static_cast<int32_t*>(pdev), static_cast<int4*>(tdev),
                               static_cast<long long*>(ndev), pool->epoch, pool->d.page_tag, s,
                               pool->exchange_ctas, nullptr, 0, timing_pair(pool, LV_TIMING_EXCHANGE),
                               nullptr, nullptr, 0, static_cast<long long*>(ndev) + 1));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

// Optional copies of a device-driven step's decisions (whole buffers: the counts
// live on the device).
cudaError_t copy_resident_outputs(lv_pool* pool, int32_t append_tokens, lv_victim* victims_out,
                                  int32_t* slots_out, int32_t* blocks_out, int32_t* pages_out,
                                  int32_t* append_out, cudaStream_t s, bool ordered = false) {
  const lv::DevPool& d = pool->d;
  const lv::ResidentScratch& rs = pool->rs;
  const struct { void* user; const void* dev; size_t bytes; } outs[] = {
      {victims_out, rs.victims, (size_t)d.budget * sizeof(lv_victim)},
      {slots_out, rs.slots, (size_t)d.budget * 4},
      {blocks_out, ordered ? rs.loads : rs.blocks, (size_t)d.maxB * 4},
      {pages_out, rs.pages, (size_t)d.maxB * 4},
      {append_out, rs.append,
       (size_t)(append_tokens / d.T + 2 < d.maxB + 2 ? append_tokens / d.T + 2 : d.maxB + 2) * 4}};
  for (const auto& o : outs) {
    if (!o.user) continue;
    const cudaError_t e = cudaMemcpyAsync(o.user, o.dev, o.bytes, cudaMemcpyDefault, s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

lv_status lv_make_resident(lv_pool* pool, int32_t sid, int64_t now_us, int32_t append_tokens,
                           uint32_t flags, int64_t max_load_pages, lv_victim* victims_out,
                           int32_t* slots_out, int32_t* blocks_out, int32_t* pages_out,
                           int32_t* append_out, lv_resident_result* result_out, lv_stream stream) {
  NvtxRange nvtx_range("lv_make_resident");
  if (!pool || sid < 0 || sid >= pool->d.S || append_tokens < 0) return LV_ERR_INVALID;
  if (flags & ~(uint32_t)(LV_RESIDENT_PRELOAD | LV_RESIDENT_ASYNC_COPY)) return LV_ERR_INVALID;
  const bool preload = (flags & LV_RESIDENT_PRELOAD) != 0;
  const bool async = (flags & LV_RESIDENT_ASYNC_COPY) != 0;
  if (preload && append_tokens != 0) return LV_ERR_INVALID;
  if (pool->d.host_pages == 0) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  const DevPool& d = pool->d;
  try {
    Staging st(pool, s);
    void* rdev = nullptr;
    lv_status r;
    if ((r = st.out(result_out, sizeof(lv_resident_result), &rdev, false)) != LV_OK) return r;
    if (++pool->epoch <= 0) pool->epoch = 1;
    const lv::ResidentScratch* rs = nullptr;
    lv::CopyOffload off{};
    LV_TRY(next_scratch(pool, s, async, &rs, &off));
    const lv::EventPair* ev = timing_pair(pool, LV_TIMING_EXCHANGE);
    auto launch = [&](cudaStream_t cs) {
      return lv::launch_make_resident(d, *rs, sid, now_us, append_tokens, preload, max_load_pages,
                                      pool->epoch, cs, pool->exchange_ctas,
                                      static_cast<lv_resident_result*>(rdev), ev, nullptr,
                                      async ? &off : nullptr);
    };
    LV_TRY(async || ev ? launch(s) : run_step(pool, s, launch));
    LV_TRY(copy_resident_outputs(pool, append_tokens, victims_out, slots_out, blocks_out, pages_out,
                                 append_out, s));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_evict(lv_pool* pool, int64_t now_us, int64_t k, uint32_t flags, lv_victim* victims_out,
                   int32_t* slots_out, lv_resident_result* result_out, lv_stream stream) {
  NvtxRange nvtx_range("lv_evict");
  if (!pool || k < 0 || (flags & ~(uint32_t)LV_RESIDENT_ASYNC_COPY)) return LV_ERR_INVALID;
  if (pool->d.host_pages == 0) return LV_ERR_INVALID;
  const bool async = (flags & LV_RESIDENT_ASYNC_COPY) != 0;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    Staging st(pool, s);
    void* rdev = nullptr;
    lv_status r;
    if ((r = st.out(result_out, sizeof(lv_resident_result), &rdev, false)) != LV_OK) return r;
    if (++pool->epoch <= 0) pool->epoch = 1;
    const lv::ResidentScratch* rs = nullptr;
    lv::CopyOffload off{};
    LV_TRY(next_scratch(pool, s, async, &rs, &off));
    const int64_t kk = k < (int64_t)pool->d.budget ? k : (int64_t)pool->d.budget;
    const lv::EventPair* ev = timing_pair(pool, LV_TIMING_EXCHANGE);
    auto launch = [&](cudaStream_t cs) {
      return lv::launch_evict(pool->d, *rs, now_us, kk, pool->epoch, cs, pool->exchange_ctas,
                              static_cast<lv_resident_result*>(rdev), ev, async ? &off : nullptr);
    };
    LV_TRY(async || ev ? launch(s) : run_step(pool, s, launch));
    LV_TRY(copy_resident_outputs(pool, 0, victims_out, slots_out, nullptr, nullptr, nullptr, s));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_join(lv_pool* pool, lv_stream stream) {
  NvtxRange nvtx_range("lv_join");
  if (!pool) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  LV_TRY(join_copies(pool, as_stream(stream)));
  return LV_OK;
}

lv_status lv_turn(lv_pool* pool, const lv_turn_desc* d, lv_victim* victims_out, int32_t* slots_out,
                  int32_t* blocks_out, int32_t* pages_out, int32_t* append_out,
                  lv_resident_result* result_out, lv_stream stream) {
  NvtxRange nvtx_range("lv_turn");
  if (!pool || !d || d->append_tokens < 0 || (d->flags & ~(uint32_t)LV_RESIDENT_ASYNC_COPY))
    return LV_ERR_INVALID;
  const bool async = (d->flags & LV_RESIDENT_ASYNC_COPY) != 0;
  if (d->sid < -1 || d->sid >= pool->d.S) return LV_ERR_INVALID;
  if (d->sid == -1 && (d->num_candidates < 1 || d->num_candidates > pool->d.S || !d->candidates))
    return LV_ERR_INVALID;
  if (pool->d.host_pages == 0) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    Staging st(pool, s);
    const void* cdev = nullptr;
    const void* kdev = nullptr;
    void* rdev = nullptr;
    lv_status r;
    if (d->sid == -1 &&
        (r = st.in(d->candidates, (size_t)d->num_candidates * 4, &cdev)) != LV_OK)
      return r;
    if (d->load_keys &&
        (r = st.in(d->load_keys, (size_t)pool->d.maxB * sizeof(uint64_t), &kdev)) != LV_OK)
      return r;
    if ((r = st.out(result_out, sizeof(lv_resident_result), &rdev, false)) != LV_OK) return r;
    if (++pool->epoch <= 0) pool->epoch = 1;
    const lv::ResidentScratch* rs = nullptr;
    lv::CopyOffload off{};
    LV_TRY(next_scratch(pool, s, async, &rs, &off));
    const lv::EventPair* ev = timing_pair(pool, LV_TIMING_EXCHANGE);
    auto launch = [&](cudaStream_t cs) {
      return lv::launch_turn(pool->d, *rs, d->sid, static_cast<const int32_t*>(cdev),
                             d->sid == -1 ? d->num_candidates : 0, d->now_us, d->append_tokens,
                             d->reply_audio_us, d->reply_units, pool->epoch, cs, pool->exchange_ctas,
                             static_cast<lv_resident_result*>(rdev), ev, async ? &off : nullptr,
                             static_cast<const unsigned long long*>(kdev));
    };
    LV_TRY(async || ev ? launch(s) : run_step(pool, s, launch));
    LV_TRY(copy_resident_outputs(pool, d->append_tokens, victims_out, slots_out, blocks_out, pages_out,
                                 append_out, s, d->load_keys != nullptr));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

namespace {
// A device address for p (device memory, or mapped page-locked host memory), else nullptr.
void* device_alias(const void* p) {
  cudaPointerAttributes a{};
  if (p == nullptr || cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) return const_cast<void*>(p);
  if (a.type == cudaMemoryTypeHost) return a.devicePointer;
  return nullptr;
}

lv_status pack_impl(lv_pool* pool, const int32_t* pages, int64_t n, void* run, bool pack, cudaStream_t s) {
  void* rdev = device_alias(run);
  if (!rdev || (reinterpret_cast<uintptr_t>(rdev) & 15)) return LV_ERR_INVALID;
  LV_TRY(join_copies(pool, s));
  Staging st(pool, s);
  const void* pin = nullptr;
  void* tdev = nullptr;
  lv_status r;
  if ((r = st.in(pages, (size_t)n * 4, &pin)) != LV_OK) return r;
  if ((r = st.out(nullptr, (size_t)n * sizeof(int4), &tdev, true)) != LV_OK) return r;
  LV_TRY(lv::launch_tasks_pages(pool->d, static_cast<const int32_t*>(pin), n, pack,
                                static_cast<int4*>(tdev), s));
  LV_TRY(lv::launch_stage(pool->d, pack, static_cast<int4*>(tdev), 0, n, static_cast<uint8_t*>(rdev), s,
                          pool->stage_ctas, timing_pair(pool, pack ? LV_TIMING_PACK : LV_TIMING_UNPACK),
                          pool->stage_tma));
  return st.finish();
}
}  // namespace

lv_status lv_pack_pages(lv_pool* pool, const int32_t* pages, int64_t n, void* dst, lv_stream stream) {
  NvtxRange nvtx_range("lv_pack_pages");
  if (!pool || n < 0 || n > 0x7fffffffll || (n > 0 && (!pages || !dst))) return LV_ERR_INVALID;
  if (n == 0) return LV_OK;
  DeviceGuard g(pool->device);
  try {
    return pack_impl(pool, pages, n, dst, true, as_stream(stream));
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_unpack_pages(lv_pool* pool, const void* src, const int32_t* pages, int64_t n,
                          lv_stream stream) {
  NvtxRange nvtx_range("lv_unpack_pages");
  if (!pool || n < 0 || n > 0x7fffffffll || (n > 0 && (!pages || !src))) return LV_ERR_INVALID;
  if (n == 0) return LV_OK;
  DeviceGuard g(pool->device);
  try {
    return pack_impl(pool, pages, n, const_cast<void*>(src), false, as_stream(stream));
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_page_checksums(lv_pool* pool, const int32_t* pages, int64_t n, uint64_t* sums_out,
                            lv_stream stream) {
  NvtxRange nvtx_range("lv_page_checksums");
  if (!pool || n < 0 || n > 0x7fffffffll || (n > 0 && (!pages || !sums_out))) return LV_ERR_INVALID;
  if (n == 0) return LV_OK;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    LV_TRY(join_copies(pool, s));   // reads KV bytes: after earlier asynchronous copies
    Staging st(pool, s);
    const void* pin = nullptr;
    void* sdev = nullptr;
    lv_status r;
    if ((r = st.in(pages, (size_t)n * 4, &pin)) != LV_OK) return r;
    if ((r = st.out(sums_out, (size_t)n * 8, &sdev, true)) != LV_OK) return r;
    void* cdev = nullptr;   // the kernel's unit cursor
    if ((r = st.out(nullptr, sizeof(unsigned long long), &cdev, true)) != LV_OK) return r;
    LV_TRY(cudaMemsetAsync(cdev, 0, sizeof(unsigned long long), s));
    LV_TRY(lv::launch_zero(sdev, n * 8, s));
    LV_TRY(lv::launch_checksums(pool->d, static_cast<const int32_t*>(pin), n,
                                static_cast<unsigned long long*>(sdev),
                                static_cast<unsigned long long*>(cdev), s, pool->num_sms * 8));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

void* lv_pool_host_device_ptr(lv_pool* pool) { return pool ? pool->d.host : nullptr; }

lv_status lv_schedule(lv_pool* pool, const lv_sched_params* q, const lv_request* reqs, int32_t n,
                      int32_t* order_out, int32_t* batch_out, lv_stream stream) {
  NvtxRange nvtx_range("lv_schedule");
  if (!pool || !q || n < 0 || n > LV_SCHED_MAX_REQUESTS || !batch_out || (n > 0 && (!reqs || !order_out)))
    return LV_ERR_INVALID;
  if (q->p_safe_us < 1 || q->p_safe_us > (1ll << 32) || q->alpha < 0 || q->alpha > (1 << 16) ||
      q->beta < 0 || q->beta > (1 << 16) || q->occupied < 0 || q->occupied > (1ll << 32) ||
      q->allocatable < 1 || q->allocatable > (1ll << 32))
    return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    Staging st(pool, s);
    const void* rin = nullptr;
    void *odev = nullptr, *bdev = nullptr;
    lv_status r;
    if ((r = st.in(reqs, (size_t)n * sizeof(lv_request), &rin)) != LV_OK) return r;
    if ((r = st.out(order_out, (size_t)n * 4, &odev, true)) != LV_OK) return r;
    if ((r = st.out(batch_out, 4, &bdev, true)) != LV_OK) return r;
    if (n == 0) {
      LV_TRY(lv::launch_zero(bdev, 4, s));
      return st.finish();
    }
    LV_TRY(lv::launch_schedule(*q, static_cast<const lv_request*>(rin), n, static_cast<int32_t*>(odev),
                               static_cast<int32_t*>(bdev), pool->d.ctl, pool->sched_scratch, s));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_remap(lv_pool* pool, const lv_remap_entry* entries, int64_t n, lv_stream stream) {
  NvtxRange nvtx_range("lv_remap");
  if (!pool || n < 0 || (n > 0 && !entries)) return LV_ERR_INVALID;
  if (n == 0) return LV_OK;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    Staging st(pool, s);
    const void* in = nullptr;
    lv_status r = st.in(entries, (size_t)n * sizeof(lv_remap_entry), &in);
    if (r != LV_OK) return r;
    if (++pool->epoch <= 0) pool->epoch = 1;
    LV_TRY(lv::launch_remap(pool->d, static_cast<const lv_remap_entry*>(in), n, pool->epoch, s,
                            pool->num_sms, pool->remap_per_thread));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_cancel(lv_pool* pool, const int32_t* locs, int64_t n, lv_stream stream) {
  NvtxRange nvtx_range("lv_cancel");
  if (!pool || n < 0 || (n > 0 && !locs)) return LV_ERR_INVALID;
  if (n == 0) return LV_OK;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    Staging st(pool, s);
    const void* in = nullptr;
    lv_status r = st.in(locs, (size_t)n * 4, &in);
    if (r != LV_OK) return r;
    LV_TRY(lv::launch_cancel(pool->d, static_cast<const int32_t*>(in), n, s));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_session_append(lv_pool* pool, int32_t sid, int32_t n_tokens, int32_t* pages_out,
                            int32_t* count_out, lv_stream stream) {
  NvtxRange nvtx_range("lv_session_append");
  if (!pool || sid < 0 || sid >= pool->d.S || n_tokens < 0) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  const size_t cap = (size_t)(n_tokens / pool->d.T) + 2;
  try {
    Staging st(pool, s);
    void *pdev = nullptr, *cdev = nullptr;
    lv_status r;
    if ((r = st.out(pages_out, cap * 4, &pdev, true)) != LV_OK) return r;
    if ((r = st.out(count_out, 4, &cdev, false)) != LV_OK) return r;
    LV_TRY(lv::launch_append(pool->d, sid, n_tokens, static_cast<int32_t*>(pdev),
                             static_cast<int32_t*>(cdev), s));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_session_counts(lv_pool* pool, int32_t* hbm_blocks, int32_t* host_blocks, lv_stream stream) {
  NvtxRange nvtx_range("lv_session_counts");
  if (!pool) return LV_ERR_INVALID;
  if (!hbm_blocks && !host_blocks) return LV_OK;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    Staging st(pool, s);
    void *a = nullptr, *b = nullptr;
    lv_status r;
    if ((r = st.out(hbm_blocks, (size_t)pool->d.S * 4, &a, false)) != LV_OK) return r;
    if ((r = st.out(host_blocks, (size_t)pool->d.S * 4, &b, false)) != LV_OK) return r;
    LV_TRY(lv::launch_counts(pool->d, static_cast<int32_t*>(a), static_cast<int32_t*>(b), s));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_session_blocks(lv_pool* pool, int32_t sid, int32_t where, int32_t* blks_out,
                            int64_t* count_out, lv_stream stream) {
  NvtxRange nvtx_range("lv_session_blocks");
  if (!pool || sid < 0 || sid >= pool->d.S || (where != 0 && where != 1) || !blks_out)
    return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  try {
    Staging st(pool, s);
    void *bdev = nullptr, *cdev = nullptr;
    lv_status r;
    if ((r = st.out(blks_out, (size_t)pool->d.maxB * 4, &bdev, true)) != LV_OK) return r;
    if ((r = st.out(count_out, 8, &cdev, false)) != LV_OK) return r;
    LV_TRY(lv::launch_blocks(pool->d, sid, where, static_cast<int32_t*>(bdev),
                             static_cast<long long*>(cdev), s));
    return st.finish();
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_read_tables(lv_pool* pool, int32_t* tables, int32_t* hbm_owner, int32_t* host_owner,
                         lv_stream stream) {
  NvtxRange nvtx_range("lv_read_tables");
  if (!pool) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  cudaStream_t s = as_stream(stream);
  const DevPool& d = pool->d;
  if (tables)
    LV_TRY(cudaMemcpyAsync(tables, d.table, (size_t)d.S * d.maxB * 4, cudaMemcpyDefault, s));
  if (hbm_owner)
    LV_TRY(cudaMemcpyAsync(hbm_owner, d.own_hbm, (size_t)d.hbm_pages * 4, cudaMemcpyDefault, s));
  if (host_owner && d.host_pages)
    LV_TRY(cudaMemcpyAsync(host_owner, d.own_host, (size_t)d.host_pages * 4, cudaMemcpyDefault, s));
  return LV_OK;
}

lv_status lv_sync(lv_pool* pool, lv_stream stream) {
  NvtxRange nvtx_range("lv_sync");
  if (!pool) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  long long ctl[2] = {0, 0};
  cudaStream_t s = as_stream(stream);
  if (join_copies(pool, s) != cudaSuccess ||
      cudaMemcpyAsync(ctl, pool->d.ctl + lv::C_ERR, sizeof(ctl), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return LV_ERR_CUDA;
  return static_cast<lv_status>(ctl[0]);
}

lv_status lv_get_stats(lv_pool* pool, lv_stats* out, lv_stream stream) {
  if (!pool || !out) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  long long c[lv::C_N];
  cudaStream_t s = as_stream(stream);
  if (cudaMemcpyAsync(c, pool->d.ctl, sizeof(c), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return LV_ERR_CUDA;
  const long long page_bytes = (long long)pool->d.J * pool->d.P;
  std::memset(out, 0, sizeof(*out));
  out->hbm_allocated = c[lv::C_HBM_ALLOC];
  out->host_allocated = c[lv::C_HOST_ALLOC];
  out->hbm_budget_pages = pool->d.budget;
  out->host_pages = pool->d.host_pages;
  out->error = c[lv::C_ERR];
  out->error_detail = c[lv::C_ERR_DETAIL];
  out->last_select_count = c[lv::C_SEL_COUNT];
  out->last_select_total = c[lv::C_SEL_TOTAL];
  out->selects = c[lv::C_SELECTS];
  out->victims = c[lv::C_VICTIMS];
  out->shortfalls = c[lv::C_SHORTFALLS];
  out->pages_out = c[lv::C_PAGES_OUT];
  out->pages_in = c[lv::C_PAGES_IN];
  out->bytes_out = (c[lv::C_PAGES_OUT] - c[lv::C_CLEAN_OUT]) * page_bytes;
  out->bytes_in = c[lv::C_PAGES_IN] * page_bytes;
  out->remap_entries = c[lv::C_REMAP];
  out->appended_pages = c[lv::C_APPENDED];
  out->cancels = c[lv::C_CANCELS];
  out->events = c[lv::C_EVENTS];
  out->fallback_selects = c[lv::C_FALLBACK];
  out->preloads = c[lv::C_PRELOADS];
  out->preloads_skipped = c[lv::C_PRELOADS_SKIPPED];
  out->clean_copies = c[lv::C_CLEAN];
  out->clean_out = c[lv::C_CLEAN_OUT];
  out->clean_dropped = c[lv::C_CLEAN_DROPPED];
  return LV_OK;
}

lv_status lv_clear_error(lv_pool* pool, lv_stream stream) {
  if (!pool) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  LV_TRY(cudaMemsetAsync(pool->d.ctl + lv::C_ERR, 0, 2 * sizeof(long long), as_stream(stream)));
  return LV_OK;
}

lv_status lv_timing_enable(lv_pool* pool, int32_t enable) {
  if (!pool) return LV_ERR_INVALID;
  pool->timing = enable != 0;
  return LV_OK;
}

lv_status lv_timing_read(lv_pool* pool, lv_kernel_timing* out, int32_t reset) {
  if (!pool || !out) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  for (int kind = 0; kind < LV_TIMING_KINDS; ++kind) {
    lv_kernel_timing t{0, 0.0, 0.0, 0.0};
    for (const lv::EventPair& e : pool->ev_used[kind]) {
      if (cudaEventSynchronize(e.end) != cudaSuccess) return LV_ERR_CUDA;
      float ms = 0.f;
      if (cudaEventElapsedTime(&ms, e.start, e.end) != cudaSuccess) return LV_ERR_CUDA;
      t.total_ms += ms;
      t.min_ms = t.launches == 0 || ms < t.min_ms ? ms : t.min_ms;
      t.max_ms = ms > t.max_ms ? ms : t.max_ms;
      t.launches += 1;
    }
    out[kind] = t;
    if (reset) {
      for (const lv::EventPair& e : pool->ev_used[kind]) pool->ev_free.push_back(e);
      pool->ev_used[kind].clear();
    }
  }
  return LV_OK;
}

lv_status lv_inject_fault(lv_pool* pool, int32_t kind, int32_t after) {
  if (!pool || kind < LV_FAULT_NONE || kind > LV_FAULT_COPY || after < 0) return LV_ERR_INVALID;
  pool->fault_kind = kind;
  pool->fault_after = after;
  return LV_OK;
}

lv_status lv_selftest_wait(lv_pool* pool, int64_t limit_us, lv_stream stream) {
  if (!pool || limit_us < 1 || limit_us > 10000000) return LV_ERR_INVALID;
  DeviceGuard g(pool->device);
  LV_TRY(lv::launch_selftest_wait(pool->d, limit_us * 1000, as_stream(stream)));
  return LV_OK;
}

const char* lv_status_str(lv_status s) {
  switch (s) {
    case LV_OK: return "LV_OK";
    case LV_ERR_INVALID: return "LV_ERR_INVALID";
    case LV_ERR_OOM: return "LV_ERR_OOM";
    case LV_ERR_CUDA: return "LV_ERR_CUDA";
    case LV_ERR_NO_HBM: return "LV_ERR_NO_HBM";
    case LV_ERR_NO_HOST: return "LV_ERR_NO_HOST";
    case LV_ERR_BOUNDS: return "LV_ERR_BOUNDS";
    case LV_ERR_DOUBLE_MAP: return "LV_ERR_DOUBLE_MAP";
    case LV_ERR_BUDGET: return "LV_ERR_BUDGET";
    case LV_ERR_TIMEOUT: return "LV_ERR_TIMEOUT";
    case LV_ERR_STATE: return "LV_ERR_STATE";
  }
  return "LV_ERR_UNKNOWN";
}

int32_t lv_version(void) { return LV_VERSION; }

}  // extern "C"
