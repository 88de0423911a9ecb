// lv_select_victims_noalloc: the victim ranker for callers that cannot allocate.
//
// Some callers must not allocate GPU memory when they rank: a serving engine
// that reserved nearly all free HBM for its KV pages at start-up (a later
// cudaMalloc can fail, or fragment that reservation), or a latency-critical
// scheduler thread (cudaMalloc and cudaFree may synchronise the device and
// stall other work).  This entry point takes the session table and block
// tables the caller already owns, and keeps its own working memory in one
// fixed array compiled into the library, so a call allocates nothing.
#include <cstdint>
#include <mutex>

#include "lv_internal.cuh"

namespace {

constexpr int kMaxSessions = LV_NOALLOC_MAX_SESSIONS;
constexpr size_t kKeyBytes = sizeof(unsigned long long) * kMaxSessions;
constexpr size_t kCountBytes = sizeof(int32_t) * kMaxSessions;
constexpr size_t kBeforeBytes = sizeof(long long) * kMaxSessions;
constexpr size_t kCtlBytes = sizeof(long long) * lv::C_N;
constexpr size_t kScratchBytes = kKeyBytes + kCountBytes + kBeforeBytes + kCtlBytes;

// The ranking scratch of every call on a device (80 KiB + 256 B).  Every GPU
// that loads liblv holds one copy until the process exits.
static __device__ __align__(256) unsigned char g_rank_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_dev[kMaxDevices] = {};

// Device address of g_rank_scratch on device `dev` (the current device), looked up
// once per device (host code cannot use the symbol itself as a device address).
// The address is kept for the life of the process: it does not survive a
// cudaDeviceReset, which lv.h tells callers.
lv_status scratch_for_device(int dev, unsigned char** out) {
  if (dev < 0 || dev >= kMaxDevices) return LV_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_dev[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_rank_scratch) != cudaSuccess || ptr == nullptr) {
      cudaGetLastError();
      return LV_ERR_CUDA;
    }
    g_scratch_dev[dev] = ptr;
  }
  *out = static_cast<unsigned char*>(g_scratch_dev[dev]);
  return LV_OK;
}

// A device address for p that device `dev` can use: device memory of that device
// as is, managed memory as is, mapped page-locked host memory through its device
// alias; anything else (pageable memory, another device's memory, page-locked
// memory with no alias) is rejected with nullptr.
const void* device_view(const void* p, int dev) {
  cudaPointerAttributes a{};
  if (p == nullptr || cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (a.type == cudaMemoryTypeDevice) return a.device == dev ? p : nullptr;
  if (a.type == cudaMemoryTypeManaged) return p;
  if (a.type == cudaMemoryTypeHost) return a.devicePointer;
  return nullptr;
}

}  // namespace

extern "C" lv_status lv_select_victims_noalloc(const lv_rank_params* prm,
                                               const lv_session_state* sessions,
                                               const int32_t* tables, int64_t now_us, int64_t k,
                                               lv_victim* out, int64_t capacity,
                                               int64_t* count_out, lv_stream stream) {
  if (!prm || prm->num_sessions < 1 || prm->num_sessions > kMaxSessions) return LV_ERR_INVALID;
  if (prm->max_blocks < 1 || prm->max_blocks > 65536 || prm->page_tokens < 1) return LV_ERR_INVALID;
  if (prm->within_order != LV_SUFFIX_FIRST && prm->within_order != LV_ASCENDING) return LV_ERR_INVALID;
  if (prm->t_play_mode != LV_PLAY_PLAYBACK && prm->t_play_mode != LV_PLAY_COUNTERS) return LV_ERR_INVALID;
  if (prm->flags & ~(uint32_t)LV_SELECT_FALLBACK) return LV_ERR_INVALID;
  if (prm->reply_prior_us < 0 || prm->unit_us < 1 || prm->unit_us > (1ll << 31)) return LV_ERR_INVALID;
  if (prm->policy != LV_POLICY_NEXT_USE && prm->policy != LV_POLICY_LRU) return LV_ERR_INVALID;
  if (prm->reserved != 0) return LV_ERR_INVALID;
  if (k < 0 || capacity < 0) return LV_ERR_INVALID;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return LV_ERR_CUDA;
  }
  const int64_t keff = k < capacity ? k : capacity;
  const void* sess = device_view(sessions, dev);
  const void* tab = device_view(tables, dev);
  void* vout = keff > 0 ? const_cast<void*>(device_view(out, dev)) : nullptr;
  void* cout = count_out ? const_cast<void*>(device_view(count_out, dev)) : nullptr;
  if (!sess || !tab || (keff > 0 && !vout) || (count_out && !cout)) return LV_ERR_INVALID;

  unsigned char* scratch = nullptr;
  lv_status st = scratch_for_device(dev, &scratch);
  if (st != LV_OK) return st;

  lv::DevPool p{};
  p.S = prm->num_sessions;
  p.maxB = prm->max_blocks;
  p.T = prm->page_tokens;
  p.within = prm->within_order;
  p.tplay = prm->t_play_mode;
  p.policy = prm->policy;
  p.reply_prior_us = prm->reply_prior_us;
  p.unit_us = prm->unit_us;
  p.sess = const_cast<lv_session_state*>(static_cast<const lv_session_state*>(sess));
  p.table = const_cast<int32_t*>(static_cast<const int32_t*>(tab));
  p.skey = reinterpret_cast<unsigned long long*>(scratch);
  p.scount = reinterpret_cast<int32_t*>(scratch + kKeyBytes);
  p.sbefore = reinterpret_cast<long long*>(scratch + kKeyBytes + kCountBytes);
  p.ctl = reinterpret_cast<long long*>(scratch + kKeyBytes + kCountBytes + kBeforeBytes);

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the counters and counts left by the previous call start again from zero;
  // keys and counts are rewritten for every session each call
  if (cudaMemsetAsync(p.ctl, 0, kCtlBytes, s) != cudaSuccess) return LV_ERR_CUDA;
  if (lv::launch_select(p, now_us, keff, (prm->flags & LV_SELECT_FALLBACK) != 0,
                        static_cast<lv_victim*>(vout), static_cast<long long*>(cout), s, 0) !=
      cudaSuccess)
    return LV_ERR_CUDA;
  return LV_OK;
}
