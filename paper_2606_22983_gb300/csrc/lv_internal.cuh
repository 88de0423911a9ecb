// Internal declarations shared by the kernels and the C-ABI layer of liblv.
#pragma once

#include <cstdint>
#include <memory>
#include <vector>
#include <cuda_runtime.h>

#include "lv.h"

namespace lv {

// Owner words: the (sid << 16 | blk) that owns a page or slot, or one of two states.
constexpr uint32_t kOwnerNone = 0xFFFFFFFFu;       // free
constexpr uint32_t kOwnerReserved = 0xFFFFFFFEu;   // reserved by a swap, not yet committed
// freed by lv_remap's commit pass; its release pass makes it kOwnerNone and clears
// the bitmap bit (no key reaches this value: sid < 4096)
constexpr uint32_t kOwnerFreeing = 0xFFFFFFFDu;
constexpr long long kKeyMax = 0xFFFFFFFFll;   // T_next is clamped to 32 bits (microseconds)

// Layout of the per-pool int64 control block in device memory.
enum Ctl : int {
  C_HBM_ALLOC = 0,     // HBM pages reserved or owned
  C_HOST_ALLOC = 1,    // host slots reserved or owned
  C_ERR = 2,           // sticky lv_status (first device-detected error)
  C_ERR_DETAIL = 3,
  C_SEL_COUNT = 4,     // victims written by the last select
  C_SEL_TOTAL = 5,     // candidates seen by the last select
  C_CLEAN = 6,         // clean host copies held now (inclusive tiers; part of C_HOST_ALLOC)
  C_RANK_TOTAL = 7,    // ranking scratch: resident blocks of all candidate sessions
  C_SELECTS = 8,
  C_VICTIMS,
  C_SHORTFALLS,
  C_PAGES_OUT,
  C_PAGES_IN,
  C_REMAP,
  C_APPENDED,
  C_CANCELS,
  C_EVENTS,
  C_FALLBACK,
  C_PRELOADS,
  C_PRELOADS_SKIPPED,
  C_CLEAN_OUT,         // evictions that found a clean copy (moved no bytes)
  C_CLEAN_DROPPED,     // clean copies dropped because their block gained rows
  C_N = 32
};

// Everything a kernel needs to know about a pool, passed by value.
struct DevPool {
  int32_t S;              // sessions
  int32_t maxB;           // block-table capacity per session
  int32_t T;              // tokens per page
  int32_t J;              // sub-pages per page (2L)
  int64_t P;              // bytes per sub-page (multiple of 16)
  int64_t hbm_pages, budget, host_pages;
  int64_t reply_prior_us, protect_us, unit_us;
  int32_t within;         // LV_SUFFIX_FIRST / LV_ASCENDING
  int32_t tplay;          // LV_PLAY_PLAYBACK / LV_PLAY_COUNTERS
  int32_t policy;         // LV_POLICY_NEXT_USE / LV_POLICY_LRU
  int32_t incl;           // 1: LV_TIERS_INCLUSIVE
  int32_t stages;         // shared-memory stages of the TMA pack/unpack kernel (0: from P)
  int32_t xstages;        // stages of the TMA exchange copy (0: the 16-byte LSU copy kernel)
  uint8_t* const* kv;     // [J] device pointers, sub-page j of page p at kv[j] + p*P
  uint8_t* host;          // device view of the host pool [host_pages][J][P]
  lv_session_state* sess; // [S]
  int32_t* table;         // [S][maxB]
  int32_t* mark;          // [S][maxB] epoch of the last remap that touched the block
  int32_t* shadow;        // [S][maxB] host slot holding the block's clean copy, or -1
  uint32_t* own_hbm;      // [hbm_pages] owner word (kOwnerNone / kOwnerReserved / sid << 16 | blk)
  uint32_t* own_host;     // [host_pages]
  uint32_t* bits_hbm;     // allocation bitmap, 1 = reserved or owned
  uint32_t* bits_host;
  long long* ctl;         // [C_N]
  // ranking scratch
  unsigned long long* skey;  // [S] session order key (0 = not a candidate)
  int32_t* scount;           // [S] resident blocks of the session
  long long* sbefore;        // [S] resident blocks of the candidates ranked ahead of it
  // exchange scratch
  unsigned long long* page_tag;  // [hbm_pages] epoch << 32 | victim index (| paired bit)
};

__host__ __device__ inline uint32_t owner_key(int32_t sid, int32_t blk) {
  return ((uint32_t)sid << 16) | ((uint32_t)blk & 0xFFFFu);   // sid < 4096, blk < 65536
}

// Optional CUDA events recorded around a copy kernel launch.
struct EventPair {
  cudaEvent_t start;
  cudaEvent_t end;
};

// Page copies moved off the caller's stream (LV_RESIDENT_ASYNC_COPY): the copy
// waits for `planned` (recorded on the caller's stream after the plan), runs on
// `stream`, and records `copied` there.
struct CopyOffload {
  cudaStream_t stream;
  cudaEvent_t planned;
  cudaEvent_t copied;
  // events recorded on `stream` just before and just after the copy kernel when the timing
  // instrument is off (it records its own pair there when on): measured, the asynchronous
  // turns run at 334-338 GB/s with a pair there (timing or not) and at 316 GB/s without one
  cudaEvent_t started;
  cudaEvent_t finished;
};

// ---- launch wrappers (lv_kernels.cu); each returns cudaGetLastError() ----
cudaError_t launch_import(const DevPool& p, const int32_t* placement, const int32_t* ctx,
                          cudaStream_t s);
cudaError_t launch_session_set(const DevPool& p, const lv_session_state* in, int32_t first,
                               int32_t n, cudaStream_t s);
cudaError_t launch_events(const DevPool& p, const lv_event* ev, int64_t n, cudaStream_t s);
cudaError_t launch_select(const DevPool& p, int64_t now_us, int64_t k, bool fallback,
                          lv_victim* out, long long* count_dev, cudaStream_t s, int num_sms,
                          const long long* k_dev = nullptr);
cudaError_t launch_alloc(const DevPool& p, bool hbm, int64_t n, int32_t* out, cudaStream_t s,
                         bool injected_fail = false);
// host slots for n victims: a clean copy where the block has one (inclusive
// tiers), else the lowest free slots in victim order (reserved)
cudaError_t launch_alloc_out(const DevPool& p, const lv_victim* v, int64_t n, int32_t* out,
                             cudaStream_t s, bool injected_fail = false);
cudaError_t launch_swap_out(const DevPool& p, const lv_victim* v, const int32_t* slots,
                            int64_t n, lv_remap_entry* commit, cudaStream_t s, int num_sms,
                            const EventPair* ev = nullptr);
cudaError_t launch_swap_in(const DevPool& p, int32_t sid, const int32_t* blks,
                           const int32_t* pages, int64_t n, lv_remap_entry* commit,
                           cudaStream_t s, int num_sms, const EventPair* ev = nullptr);
cudaError_t launch_exchange(const DevPool& p, const lv_victim* v, int64_t n_out, int32_t sid,
                            const int32_t* blks, int64_t n_in, int32_t* slots, int32_t* pages,
                            int4* tasks, long long* n_tasks, int32_t epoch,
                            unsigned long long* page_tag, cudaStream_t s, int copy_ctas,
                            const long long* counts_dev = nullptr, long long max_units = 0,
                            const EventPair* ev = nullptr, const long long* sid_dev = nullptr,
                            const CopyOffload* off = nullptr, int gate = 0,
                            long long* cursor = nullptr, const struct StepFinish* fin = nullptr);
cudaError_t launch_remap(const DevPool& p, const lv_remap_entry* e, int64_t n, int32_t epoch,
                         cudaStream_t s, int num_sms, int per_thread);
cudaError_t launch_cancel(const DevPool& p, const int32_t* locs, int64_t n, cudaStream_t s);
// Zeroes bytes (a multiple of 4) at q: device memory or mapped page-locked host memory.
cudaError_t launch_zero(void* q, int64_t bytes, cudaStream_t s);
// fin (with R, the step's control words): a device-driven step's end, done by the
// append kernel after the growth
cudaError_t launch_append(const DevPool& p, int32_t sid, int32_t n_tokens, int32_t* pages,
                          int32_t* count, cudaStream_t s, const long long* gate = nullptr,
                          const long long* sid_dev = nullptr, const struct StepFinish* fin = nullptr,
                          const long long* R = nullptr);

// One kernel launch of a device-driven step, recorded instead of issued (for replay
// through a CUDA graph): the kernel, its launch shape, whether it is a programmatic
// dependent launch, and its argument values (`args` points into `holder`).
struct LaunchRecord {
  const void* func;
  dim3 grid, block;
  size_t smem;
  bool pdl;
  std::shared_ptr<void> holder;
  std::vector<void*> args;
};
// While a recorder is set on the calling host thread, the step launchers append their
// programmatic dependent launches to it instead of issuing them.
void set_launch_recorder(std::vector<LaunchRecord>* rec);
// Issues recorded launches on s (the same launches the launchers would have made).
cudaError_t replay_launches(const std::vector<LaunchRecord>& recs, cudaStream_t s);

// Device buffers of lv_make_resident, owned by the pool.
struct ResidentScratch {
  lv_victim* victims;   // [budget]
  int32_t* slots;       // [budget]
  int32_t* blocks;      // [maxB] the session's host-tier blocks, ascending
  int32_t* loads;       // [maxB] the same blocks in the caller's load order (load keys)
  int32_t* pages;       // [maxB]
  int32_t* append;      // [maxB + 2]
  int4* tasks;          // [budget + maxB]
  long long* words;     // [16]
  int32_t* hits;        // [S] lv_turn's pick
};
// The end of a device-driven step (lv_make_resident, lv_turn, lv_evict): the turn's
// LV_EV_TURN_END, a completed preload's protection, and the result record.
struct StepFinish {
  bool on;
  int32_t sid;                    // the session, or read from sid_dev when that is set
  const long long* sid_dev;
  long long now_us;
  bool preload;
  bool turn_end;
  long long audio_us, units;      // LV_EV_TURN_END's a and b
  lv_resident_result* out;        // may be null
};
// lv_turn's start, done by the first kernel of the make-resident chain: pick the
// session when sid < 0 (the first of cand[0..n_cand) with hit set), then TURN_BEGIN.
struct TurnStart {
  bool on;
  const int32_t* cand;
  int32_t n_cand;
  const int32_t* hit;
  long long now_us;
};
cudaError_t launch_make_resident(const DevPool& p, const ResidentScratch& rs, int32_t sid,
                                 int64_t now_us, int32_t append_tokens, bool preload,
                                 int64_t max_load, int32_t epoch, cudaStream_t s, int copy_ctas,
                                 lv_resident_result* result, const EventPair* ev = nullptr,
                                 const long long* sid_dev = nullptr, const CopyOffload* off = nullptr,
                                 const unsigned long long* load_keys = nullptr, bool turn_end = false,
                                 int64_t audio_us = 0, int64_t units = 0,
                                 const TurnStart* ts = nullptr);
// lv_turn: pick (sid < 0), LV_EV_TURN_BEGIN, make resident, LV_EV_TURN_END
// lv_evict: rank, evict up to k victims (no loads), finish
cudaError_t launch_evict(const DevPool& p, const ResidentScratch& rs, int64_t now_us, int64_t k,
                         int32_t epoch, cudaStream_t s, int copy_ctas, lv_resident_result* result,
                         const EventPair* ev, const CopyOffload* off);
cudaError_t launch_turn(const DevPool& p, const ResidentScratch& rs, int32_t sid, const int32_t* cand,
                        int32_t n_cand, int64_t now_us, int32_t append_tokens, int64_t audio_us,
                        int64_t units, int32_t epoch, cudaStream_t s, int copy_ctas,
                        lv_resident_result* result, const EventPair* ev = nullptr,
                        const CopyOffload* off = nullptr, const unsigned long long* load_keys = nullptr);
cudaError_t launch_counts(const DevPool& p, int32_t* hbm, int32_t* host, cudaStream_t s);
// sums[i] = position-weighted 64-bit sum of page pages[i] (sums zeroed by the caller)
cudaError_t launch_checksums(const DevPool& p, const int32_t* pages, int64_t n,
                             unsigned long long* sums, unsigned long long* cursor, cudaStream_t s,
                             int ctas);
cudaError_t launch_blocks(const DevPool& p, int32_t sid, int32_t where, int32_t* out,
                          long long* count, cudaStream_t s);
cudaError_t launch_check_budget(const DevPool& p, cudaStream_t s);
// staged path
cudaError_t launch_tasks_out(const DevPool& p, const lv_victim* v, const int32_t* slots, int64_t n,
                             int4* tasks, lv_remap_entry* commit, cudaStream_t s);
cudaError_t launch_tasks_in(const DevPool& p, int32_t sid, const int32_t* blks, const int32_t* pages,
                            int64_t n, int4* tasks, lv_remap_entry* commit, cudaStream_t s);
cudaError_t launch_exchange_plan(const DevPool& p, const lv_victim* v, int64_t n_out, int32_t sid,
                                 const int32_t* blks, int64_t n_in, int32_t* slots, int32_t* pages,
                                 int4* tasks, long long* n_tasks, int32_t epoch,
                                 unsigned long long* page_tag, cudaStream_t s);
// pack (staging[t] <- out pages) or unpack (in pages <- staging[t]) for tasks [t_begin, t_end)
cudaError_t launch_stage(const DevPool& p, bool pack, const int4* tasks, int64_t t_begin,
                         int64_t t_end, uint8_t* staging, cudaStream_t s, int ctas,
                         const EventPair* ev, bool tma);
cudaError_t launch_tasks_pages(const DevPool& p, const int32_t* pages, int64_t n, bool pack,
                               int4* tasks, cudaStream_t s);
cudaError_t configure_stage_kernels(const DevPool& p);
// The largest number of exchange-copy TMA stages (2P bytes each) for sub-pages of P
// bytes (0 when two do not fit in a CTA's shared memory), and the kernel's set-up.
int exchange_stage_limit(long long P);
cudaError_t configure_exchange_tma(const DevPool& p);
cudaError_t launch_selftest_wait(const DevPool& p, long long limit_ns, cudaStream_t s);
// lv_sched.cu
// scratch: device memory of 32 * LV_SCHED_MAX_REQUESTS bytes (keys and costs)
cudaError_t launch_schedule(const lv_sched_params& q, const lv_request* reqs, int n, int32_t* order,
                            int32_t* batch, long long* ctl, void* scratch, cudaStream_t s);
// lv_api.cu: the shape of a pool (for the controller)
void pool_shape(const lv_pool* pool, int32_t* sessions, int32_t* max_blocks, int64_t* page_bytes,
                int64_t* budget, int64_t* host_pages);

}  // namespace lv
