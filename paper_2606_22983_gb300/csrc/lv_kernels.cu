// CUDA kernels of the KV swap path (sm_103a).
//
//   ranking   k_rank_census -> k_rank_emit                (Section 5.1, Eq. 4)
//   allocate  k_alloc, k_alloc_out                           (lowest free, Section 5.1)
//   move      k_swap_out / k_swap_in                         (Section 5, Fig. 6; Section 5.2)
//             k_exchange_plan -> k_exchange_copy             (both directions in one step)
//             k_stage_tasks (TMA) / k_stage_tasks_lsu         (staged copy-engine path)
//   commit    k_remap, k_cancel, k_append                    (Section 6 side tables)
//   monitor   k_events                                       (Section 3, Sections 5.1-5.2)
//   turn      k_resident_*, k_pick_scan,                      (a whole turn on the device;
//             k_order_loads, k_evict_prepare                 the gate runs in the plan)
//   verify    k_checksum                                     (page checksums)
//
// The only waits are the TMA stage kernel's mbarrier waits for its own copies,
// each limited by %globaltimer to one second, after which the kernel reports
// LV_ERR_TIMEOUT and returns; no kernel waits on another kernel or agent.  Every
// index read from memory is range-checked and a bad item is skipped with the
// sticky error set.
#include <cstdint>
#include <memory>
#include <tuple>
#include <utility>

#include "lv_internal.cuh"

namespace lv {

namespace {

__device__ __forceinline__ void set_error(long long* ctl, int code, long long detail) {
  if (atomicCAS(reinterpret_cast<unsigned long long*>(&ctl[C_ERR]), 0ull,
                (unsigned long long)code) == 0ull) {
    ctl[C_ERR_DETAIL] = detail;
  }
}

// Programmatic dependent launch.  The kernels of a device-driven step are
// launched so that each may be scheduled while the previous kernel on the
// stream still runs (its launch latency overlaps that kernel).  Each of them
// begins with pdl_entry(): it waits until the previous kernel has completed
// and its writes are visible -- nothing of the kernel runs earlier -- and then
// lets the next kernel of the stream be scheduled.  In a kernel launched the
// ordinary way both instructions have no effect.
__device__ __forceinline__ void pdl_entry() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// The same two steps apart, for a kernel with a large grid: it waits at its start and
// lets the next kernel be scheduled only when its own work is done, so that the next
// kernel's CTAs do not sit on SMs, waiting, while this grid still needs them.  A CTA
// that returns early counts as having let it.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ int32_t nblocks_of(const DevPool& p, int32_t sid) {
  long long c = p.sess[sid].ctx_tokens;
  long long nb = (c + p.T - 1) / p.T;
  if (nb < 0) nb = 0;
  if (nb > p.maxB) nb = p.maxB;
  return (int32_t)nb;
}

// Exclusive scan over the block of NT threads; *total receives the sum.
template <int NT>
__device__ long long block_excl_scan(long long v, long long* total) {
  static_assert(NT % 32 == 0 && NT <= 1024, "block size");
  __shared__ long long warp_sums[NT / 32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  long long x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    long long y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[wid] = x;
  __syncthreads();
  if (wid == 0) {
    long long w = lane < NT / 32 ? warp_sums[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      long long y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < NT / 32) warp_sums[lane] = w;
  }
  __syncthreads();
  long long before = wid > 0 ? warp_sums[wid - 1] : 0;
  *total = warp_sums[NT / 32 - 1];
  __syncthreads();
  return before + x - v;
}

__device__ __forceinline__ uint32_t free_bits(const uint32_t* bits, long long w, long long W,
                                              long long nbits) {
  uint32_t valid = 0xffffffffu;
  if (w == W - 1 && (nbits & 31)) valid = (1u << (nbits & 31)) - 1u;
  return ~bits[w] & valid;
}

// The n lowest free bits of a bitmap, ascending, into out[0..n); sets them.
// Each thread owns a contiguous run of words and writes only the ranks it
// counted, so a concurrent free elsewhere cannot make two threads write one rank.
template <int NT>
__device__ void block_alloc_lowest(uint32_t* bits, long long nbits, long long n, int32_t* out) {
  const long long W = (nbits + 31) >> 5;
  const long long per = (W + NT - 1) / NT;
  const long long w0 = min(W, (long long)threadIdx.x * per);
  const long long w1 = min(W, w0 + per);
  long long cnt = 0;
  for (long long w = w0; w < w1; ++w) cnt += __popc(free_bits(bits, w, W, nbits));
  long long total;
  const long long base = block_excl_scan<NT>(cnt, &total);
  long long r = base;
  const long long r_end = min(n, base + cnt);
  for (long long w = w0; w < w1 && r < r_end; ++w) {
    uint32_t f = free_bits(bits, w, W, nbits);
    uint32_t take = 0;
    while (f && r < r_end) {
      int b = __ffs(f) - 1;
      f &= f - 1;
      out[r++] = (int32_t)(w * 32 + b);
      take |= 1u << b;
    }
    if (take) atomicOr(&bits[w], take);
  }
}

// Inclusive tiers: the host slot holding victim x's clean copy, or -1.
__device__ __forceinline__ int32_t clean_copy_of(const DevPool& p, const lv_victim& x) {
  if (!p.incl || x.sid < 0 || x.sid >= p.S || x.blk < 0 || x.blk >= p.maxB) return -1;
  return p.shadow[(size_t)x.sid * p.maxB + x.blk];
}

// Host slots for n victims when nd of them have no clean copy: the nd lowest
// free slots are taken (ascending) into out[0..nd), then spread in place so
// that the r-th victim without a copy gets the r-th slot and every other
// victim its copy.  The spreading runs from the last chunk to the first: a
// victim's rank r is at most its index, so each read position still holds its
// compact value when it is read.
template <int NT>
__device__ void block_alloc_out(const DevPool& p, const lv_victim* __restrict__ v, long long n,
                                long long nd, int32_t* out) {
  if (nd > 0) block_alloc_lowest<NT>(p.bits_host, p.host_pages, nd, out);
  __syncthreads();
  for (long long r = threadIdx.x; r < nd; r += NT) p.own_host[out[r]] = kOwnerReserved;
  __syncthreads();
  if (nd == n) return;
  long long after = 0;   // victims without a copy in the chunks already spread
  for (long long c = (n + NT - 1) / NT - 1; c >= 0; --c) {
    const long long i = c * NT + threadIdx.x;
    int32_t cp = -1;
    long long d = 0;
    if (i < n) {
      cp = clean_copy_of(p, v[i]);
      d = cp < 0;
    }
    long long chunk;
    const long long excl = block_excl_scan<NT>(d, &chunk);
    const int32_t val = (i < n && d) ? out[nd - after - chunk + excl] : cp;
    __syncthreads();
    if (i < n) out[i] = val;
    __syncthreads();
    after += chunk;
  }
}

// ---------------------------------------------------------------- import
__global__ void k_import(DevPool p, const int32_t* __restrict__ placement,
                         const int32_t* __restrict__ ctx) {
  const long long total = (long long)p.S * p.maxB;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
       idx += (long long)gridDim.x * blockDim.x) {
    const int32_t s = (int32_t)(idx / p.maxB), b = (int32_t)(idx % p.maxB);
    const long long c = ctx[s];
    long long nb = (c + p.T - 1) / p.T;
    if (b == 0) {
      if (c < 0 || nb > p.maxB) {
        set_error(p.ctl, LV_ERR_BOUNDS, s);
      }
      p.sess[s].ctx_tokens = (c < 0 || nb > p.maxB) ? 0 : (int32_t)c;
    }
    if (c < 0 || nb > p.maxB) nb = 0;
    const int32_t e = placement[idx];
    p.table[idx] = -1;
    p.mark[idx] = 0;
    p.shadow[idx] = -1;
    if (b >= nb) {
      if (e != -1) set_error(p.ctl, LV_ERR_BOUNDS, idx);
      continue;
    }
    const uint32_t key = owner_key(s, b);
    if (e >= 0) {
      if (e >= p.hbm_pages) { set_error(p.ctl, LV_ERR_BOUNDS, idx); continue; }
      if (atomicCAS(&p.own_hbm[e], kOwnerNone, key) != kOwnerNone) {
        set_error(p.ctl, LV_ERR_DOUBLE_MAP, idx);
        continue;
      }
      atomicOr(&p.bits_hbm[e >> 5], 1u << (e & 31));
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_HBM_ALLOC]), 1ull);
    } else if (e <= -2) {
      const long long h = -(long long)e - 2;
      if (h >= p.host_pages) { set_error(p.ctl, LV_ERR_BOUNDS, idx); continue; }
      if (atomicCAS(&p.own_host[h], kOwnerNone, key) != kOwnerNone) {
        set_error(p.ctl, LV_ERR_DOUBLE_MAP, idx);
        continue;
      }
      atomicOr(&p.bits_host[h >> 5], 1u << (h & 31));
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_HOST_ALLOC]), 1ull);
    } else {
      set_error(p.ctl, LV_ERR_BOUNDS, idx);   // a block inside the context with no location
      continue;
    }
    p.table[idx] = e;
  }
}

__global__ void k_check_budget(DevPool p) {
  if (p.ctl[C_HBM_ALLOC] > p.budget) set_error(p.ctl, LV_ERR_BUDGET, p.ctl[C_HBM_ALLOC]);
}

// -------------------------------------------------------------- sessions
__global__ void k_session_set(DevPool p, const lv_session_state* __restrict__ in, int32_t first,
                              int32_t n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  lv_session_state st = in[i];
  st.ctx_tokens = p.sess[first + i].ctx_tokens;   // owned by import / append
  p.sess[first + i] = st;
}

// One monitor event applied to a session's state (Section 3 signals; Section
// 5.1 reply interval and immediate reuse; Section 5.2 protection).
__device__ __forceinline__ void apply_event(const DevPool& p, lv_session_state& st, const lv_event& x) {
  switch (x.kind) {
    case LV_EV_TURN_BEGIN:
      st.flags = (st.flags | LV_RUNNING) & ~LV_IMMEDIATE;
      st.protect_until_us = 0;
      st.last_use_us = x.t_us;
      break;
    case LV_EV_TURN_END:
      st.last_use_us = x.t_us;
      st.flags &= ~(LV_RUNNING | LV_DONE_VALID);
      st.gen_us = x.a;
      st.play_us = 0;
      st.reply_tokens = x.b;
      if (st.gen_us > 0) {
        st.flags |= LV_RESP_OPEN;
      } else {
        st.flags = (st.flags & ~LV_RESP_OPEN) | LV_DONE_VALID;
        st.t_done_us = x.t_us;
      }
      break;
    case LV_EV_PLAYBACK:
      if (st.flags & LV_RESP_OPEN) {
        const long long np = st.play_us + x.a;
        st.play_us = np < st.gen_us ? np : st.gen_us;
        if (st.play_us >= st.gen_us) {
          st.flags = (st.flags & ~LV_RESP_OPEN) | LV_DONE_VALID;
          st.t_done_us = x.t_us;
        }
      }
      break;
    case LV_EV_SPEECH_START:
      st.flags |= LV_IMMEDIATE;
      break;
    case LV_EV_BARGE_IN:
      st.gen_us = st.play_us;
      st.flags = (st.flags | LV_IMMEDIATE) & ~(LV_RESP_OPEN | LV_DONE_VALID);
      break;
    case LV_EV_SPEECH_STOP:
      if (st.flags & LV_DONE_VALID) {
        long long xs = x.t_us - st.t_done_us;
        if (xs < 0) xs = 0;
        st.reply_ema_us = st.reply_n == 0 ? xs : (3 * st.reply_ema_us + xs) / 4;
        if (st.reply_n < 0x7fffffff) st.reply_n += 1;
      }
      st.flags &= ~(LV_IMMEDIATE | LV_DONE_VALID);
      break;
    case LV_EV_PRELOADED:
      st.protect_until_us = x.t_us + p.protect_us;
      break;
    case LV_EV_UNPROTECT:
      st.protect_until_us = 0;
      break;
    default:
      break;   // reported by the caller
  }
}

// One thread per session applies, in order, the events addressed to it.
constexpr int kEventThreads = 128;
constexpr int kEventChunk = 512;   // events staged in shared memory at a time (16 KiB)

// One thread per session.  The CTA stages the event list in shared memory, a
// chunk at a time (coalesced loads, each event read once per CTA), and every
// thread applies, in list order, the events of its own session.  CTA 0 checks
// every event's kind and session and counts them.
__global__ void __launch_bounds__(kEventThreads)
k_events(DevPool p, const lv_event* __restrict__ ev, long long n) {
  __shared__ lv_event chunk[kEventChunk];
  const int s = blockIdx.x * kEventThreads + threadIdx.x;
  lv_session_state st;
  if (s < p.S) st = p.sess[s];
  bool touched = false;
  for (long long c0 = 0; c0 < n; c0 += kEventChunk) {
    const int m = (int)(n - c0 < kEventChunk ? n - c0 : kEventChunk);
    __syncthreads();   // the previous chunk is no longer read
    for (int e = threadIdx.x; e < m; e += kEventThreads) {
      const lv_event x = ev[c0 + e];
      chunk[e] = x;
      if (blockIdx.x == 0 && (x.kind < LV_EV_TURN_BEGIN || x.kind > LV_EV_UNPROTECT || x.sid < 0 ||
                              x.sid >= p.S))
        set_error(p.ctl, LV_ERR_BOUNDS, c0 + e);
    }
    __syncthreads();
    if (s < p.S) {
      for (int e = 0; e < m; ++e) {
        if (chunk[e].sid != s) continue;
        touched = true;
        apply_event(p, st, chunk[e]);
      }
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0)
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_EVENTS]), (unsigned long long)n);
  if (s < p.S && touched) p.sess[s] = st;
}

// --------------------------------------------------------------- ranking
// Order key of a session, 0 when it is not a candidate.  Larger keys are
// evicted first: bit 63 = normal tier, bits 31..62 = T_next (Eq. 4), bits
// 0..30 = 2^31-1-sid so that equal T_next rank by ascending session id.
__device__ __forceinline__ unsigned long long session_key(const DevPool& p, int32_t s,
                                                          long long now_us, bool fallback) {
  const lv_session_state st = p.sess[s];
  if (p.policy == LV_POLICY_LRU) {
    // least recently used first: every non-running session is a candidate
    if (st.flags & LV_RUNNING) return 0ull;
    long long t = st.last_use_us;
    if (t < 0) t = 0;
    if (t > kKeyMax) t = kKeyMax;
    return (1ull << 63) | ((unsigned long long)(kKeyMax - t) << 31) |
           (unsigned long long)(0x7fffffff - s);
  }
  const bool normal = !(st.flags & (LV_RUNNING | LV_IMMEDIATE)) && !(now_us < st.protect_until_us);
  if (!normal && !(fallback && !(st.flags & LV_RUNNING))) return 0ull;
  long long t_play;
  if (p.tplay == LV_PLAY_PLAYBACK) {
    const long long d = st.gen_us - st.play_us;            // remaining playback horizon
    t_play = d > 0 ? d : 0;
  } else {
    // progress counters: a longer unfinished reply means later reuse
    if (!(st.flags & LV_RESP_OPEN) || st.reply_tokens <= 0) t_play = 0;
    else if (st.reply_tokens > kKeyMax / p.unit_us) t_play = kKeyMax;
    else t_play = st.reply_tokens * p.unit_us;
  }
  long long t_reply = st.reply_n > 0 ? st.reply_ema_us : p.reply_prior_us;
  if (t_reply < 0) t_reply = 0;
  if (t_play > kKeyMax) t_play = kKeyMax;
  if (t_reply > kKeyMax) t_reply = kKeyMax;
  long long t_next = t_play + t_reply;
  if (t_next > kKeyMax) t_next = kKeyMax;
  return ((normal ? 1ull : 0ull) << 63) | ((unsigned long long)t_next << 31) |
         (unsigned long long)(0x7fffffff - s);
}

constexpr int kCensusThreads = 256;
// Up to this many sessions every emit CTA finds its session's place by reading all
// S keys itself (S^2 key reads, from L2); above it, k_rank_prefix computes every place
// once, between the census and the emission (S^2 key comparisons, but S^2 / 256 key
// reads), at the cost of one more launch in the chain.
#ifndef LV_EMIT_SCAN_MAX
#define LV_EMIT_SCAN_MAX 1024
#endif
constexpr int kEmitScanMax = LV_EMIT_SCAN_MAX;

// One CTA per session: its key and its count of HBM-resident blocks.
__global__ void __launch_bounds__(kCensusThreads)
k_rank_census(DevPool p, long long now_us, bool fallback, const long long* __restrict__ k_dev) {
  pdl_wait();
  if (k_dev && *k_dev == 0) return;   // a device-driven step with no deficit ranks nothing
  const int32_t s = blockIdx.x;
  __shared__ unsigned long long key;
  if (threadIdx.x == 0) {
    key = session_key(p, s, now_us, fallback);
    if (p.S > kEmitScanMax) {       // k_rank_prefix accumulates into these
      p.sbefore[s] = 0;
      if (s == 0) p.ctl[C_RANK_TOTAL] = 0;
    }
  }
  __syncthreads();
  if (key == 0ull) {
    if (threadIdx.x == 0) { p.skey[s] = 0ull; p.scount[s] = 0; }
    return;
  }
  const int32_t nb = nblocks_of(p, s);
  const int32_t* row = p.table + (size_t)s * p.maxB;
  long long c = 0;
  for (int32_t b = threadIdx.x; b < nb; b += kCensusThreads) c += row[b] >= 0 ? 1 : 0;
  long long total;
  block_excl_scan<kCensusThreads>(c, &total);
  if (threadIdx.x == 0) {
    p.skey[s] = key;
    p.scount[s] = (int32_t)total;
  }
  pdl_trigger();
}

constexpr int kPrefixTile = 128;    // sessions placed by one CTA (one per thread)
constexpr int kPrefixChunk = 256;   // keys staged by one CTA in shared memory

// The place of every candidate session in the victim order, for S > kEmitScanMax:
// sbefore[s] = the resident blocks of the candidate sessions with a larger key
// (keys are distinct).  CTA (x, y) compares the sessions of tile x with the keys
// of chunk y, read once into shared memory (every thread reads the same key at
// once: a broadcast), and adds its partial sums; the CTAs of tile 0 also add up
// all candidates' blocks into C_RANK_TOTAL.  The census zeroed both.
__global__ void __launch_bounds__(kPrefixTile)
k_rank_prefix(DevPool p, const long long* __restrict__ k_dev) {
  pdl_wait();   // the census is complete and visible
  if (k_dev && *k_dev == 0) return;
  __shared__ unsigned long long kc[kPrefixChunk];
  __shared__ int32_t cc[kPrefixChunk];
  __shared__ long long part[kPrefixTile / 32];
  const int32_t j0 = blockIdx.y * kPrefixChunk;
  const int32_t nj = min(kPrefixChunk, p.S - j0);
  for (int32_t j = threadIdx.x; j < nj; j += kPrefixTile) {
    const unsigned long long kj = p.skey[j0 + j];
    kc[j] = kj;
    cc[j] = kj ? p.scount[j0 + j] : 0;
  }
  __syncthreads();
  const int32_t s = blockIdx.x * kPrefixTile + threadIdx.x;
  const unsigned long long key = s < p.S ? p.skey[s] : 0ull;
  if (key != 0ull) {
    long long before = 0;
#pragma unroll 8
    for (int32_t j = 0; j < nj; ++j) before += kc[j] > key ? cc[j] : 0;
    if (before) atomicAdd(reinterpret_cast<unsigned long long*>(&p.sbefore[s]), (unsigned long long)before);
  }
  if (blockIdx.x == 0) {
    long long t = 0;
    for (int32_t j = threadIdx.x; j < nj; j += kPrefixTile) t += cc[j];
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = t;
    __syncthreads();
    if (threadIdx.x == 0) {
      long long all = 0;
      for (int w = 0; w < kPrefixTile / 32; ++w) all += part[w];
      if (all) atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_RANK_TOTAL]), (unsigned long long)all);
    }
  }
  pdl_trigger();
}

constexpr int kEmitThreads = 256;

// One CTA per session.  The victim order takes the sessions by decreasing key
// (keys are distinct: each holds its session id), so a session's first
// position in the order is the number of resident blocks of the sessions with
// a larger key; the CTA sums those counts over the census, then writes its
// own resident blocks, suffix first (or ascending), while positions stay below
// the selection count min(k, all resident candidates).  CTA 0 publishes the
// count and the counters.
__global__ void __launch_bounds__(kEmitThreads)
k_rank_emit(DevPool p, long long k, const long long* k_dev, bool fallback, long long* count_dev,
            lv_victim* __restrict__ out) {
  pdl_wait();   // the census (and the places) are complete and visible
  const int32_t sid = blockIdx.x;
  if (k_dev) {            // k decided on the device (lv_make_resident, lv_evict)
    k = *k_dev;
    if (k == 0) {         // no deficit: the census did not run, nothing is selected
      if (sid == 0 && threadIdx.x == 0) {
        p.ctl[C_SEL_COUNT] = 0;
        atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_SELECTS]), 1ull);
        if (fallback) atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_FALLBACK]), 1ull);
        if (count_dev) *count_dev = 0;
      }
      return;
    }
  }
  const unsigned long long key = p.skey[sid];
  if (key == 0ull && sid != 0) return;
  long long off, total;
  if (p.S > kEmitScanMax) {      // placed by k_rank_prefix
    off = key ? p.sbefore[sid] : 0;
    total = p.ctl[C_RANK_TOTAL];
  } else {
    long long before = 0, all = 0;
    for (int32_t j = threadIdx.x; j < p.S; j += kEmitThreads) {
      const unsigned long long kj = p.skey[j];
      const long long cj = kj ? p.scount[j] : 0;
      all += cj;
      before += kj > key ? cj : 0;
    }
    block_excl_scan<kEmitThreads>(before, &off);
    block_excl_scan<kEmitThreads>(all, &total);
  }
  const long long n_out = k < total ? k : total;
  if (sid == 0 && threadIdx.x == 0) {
    p.ctl[C_SEL_COUNT] = n_out;
    p.ctl[C_SEL_TOTAL] = total;
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_SELECTS]), 1ull);
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_VICTIMS]), (unsigned long long)n_out);
    if (k != INT64_MAX && total < k)
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_SHORTFALLS]), 1ull);
    if (fallback) atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_FALLBACK]), 1ull);
    if (count_dev) *count_dev = n_out;
  }
  if (key == 0ull || off >= n_out) return;
  const int32_t nb = nblocks_of(p, sid);
  const int32_t* row = p.table + (size_t)sid * p.maxB;
  const bool suffix = p.within == LV_SUFFIX_FIRST;
  long long run = 0;
  for (int32_t q0 = 0; q0 < nb && off + run < n_out; q0 += kEmitThreads) {
    const int32_t q = q0 + threadIdx.x;
    const int32_t b = suffix ? nb - 1 - q : q;
    int32_t e = -1;
    if (q < nb) e = row[b];
    const long long flag = e >= 0 ? 1 : 0;
    long long chunk;
    const long long pos = off + run + block_excl_scan<kEmitThreads>(flag, &chunk);
    if (flag && pos < n_out) out[pos] = lv_victim{sid, b, e};
    run += chunk;
  }
  pdl_trigger();
}

// ------------------------------------------------------------ allocation
constexpr int kAllocThreads = 1024;

__global__ void __launch_bounds__(kAllocThreads)
k_alloc(DevPool p, bool hbm, long long n, int32_t* __restrict__ out, bool injected_fail) {
  __shared__ int ok;
  uint32_t* bits = hbm ? p.bits_hbm : p.bits_host;
  const long long nbits = hbm ? p.hbm_pages : p.host_pages;
  const long long cap = hbm ? p.budget : p.host_pages;
  long long* counter = &p.ctl[hbm ? C_HBM_ALLOC : C_HOST_ALLOC];
  if (threadIdx.x == 0) {
    const long long before = (long long)atomicAdd(reinterpret_cast<unsigned long long*>(counter),
                                                  (unsigned long long)n);
    ok = before + n <= cap && !injected_fail;
    if (!ok) {
      atomicAdd(reinterpret_cast<unsigned long long*>(counter), (unsigned long long)(-n));
      set_error(p.ctl, hbm ? LV_ERR_NO_HBM : LV_ERR_NO_HOST, n);
    }
  }
  __syncthreads();
  if (!ok) {
    for (long long i = threadIdx.x; i < n; i += kAllocThreads) out[i] = -1;
    return;
  }
  block_alloc_lowest<kAllocThreads>(bits, nbits, n, out);
  __syncthreads();
  uint32_t* own = hbm ? p.own_hbm : p.own_host;
  for (long long i = threadIdx.x; i < n; i += kAllocThreads) own[out[i]] = kOwnerReserved;
}

// Host slots of a swap-out under inclusive tiers (one CTA): victims with a clean
// copy take it; only the others count against the host tier and reserve slots.
__global__ void __launch_bounds__(kAllocThreads)
k_alloc_out(DevPool p, const lv_victim* __restrict__ v, long long n, int32_t* __restrict__ out,
            bool injected_fail) {
  __shared__ int ok;
  __shared__ long long nd_s;
  long long cnt = 0;
  for (long long i = threadIdx.x; i < n; i += kAllocThreads) cnt += clean_copy_of(p, v[i]) < 0;
  long long nd;
  block_excl_scan<kAllocThreads>(cnt, &nd);
  if (threadIdx.x == 0) {
    long long* counter = &p.ctl[C_HOST_ALLOC];
    const long long before = (long long)atomicAdd(reinterpret_cast<unsigned long long*>(counter),
                                                  (unsigned long long)nd);
    ok = before + nd <= p.host_pages && !injected_fail;
    if (!ok) {
      atomicAdd(reinterpret_cast<unsigned long long*>(counter), (unsigned long long)(-nd));
      set_error(p.ctl, LV_ERR_NO_HOST, nd);
    }
    nd_s = nd;
  }
  __syncthreads();
  if (!ok) {
    for (long long i = threadIdx.x; i < n; i += kAllocThreads) out[i] = -1;
    return;
  }
  block_alloc_out<kAllocThreads>(p, v, n, nd_s, out);
}

// ------------------------------------------------------------------ copy
constexpr int kCopyThreads = 256;
constexpr int kCopyUnroll = 4;

// Copies one sub-page: 16-byte vectors, kCopyUnroll loads in flight per thread.
__device__ __forceinline__ void copy_subpage(const int4* __restrict__ src, int4* __restrict__ dst,
                                             int nvec) {
  for (int base = threadIdx.x; base < nvec; base += kCopyThreads * kCopyUnroll) {
    int4 r[kCopyUnroll];
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) {
      const int q = base + u * kCopyThreads;
      if (q < nvec) r[u] = src[q];
    }
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) {
      const int q = base + u * kCopyThreads;
      if (q < nvec) dst[q] = r[u];
    }
  }
}

// Unit u = (victim i, sub-page j): hbm_kv[j][page_i] -> host[slot_i][j].
__global__ void __launch_bounds__(kCopyThreads)
k_swap_out(DevPool p, const lv_victim* __restrict__ v, const int32_t* __restrict__ slots,
           long long n, lv_remap_entry* __restrict__ commit) {
  const long long units = n * p.J;
  const int nvec = (int)(p.P >> 4);
  for (long long u = blockIdx.x; u < units; u += gridDim.x) {
    const long long i = u / p.J;
    const int j = (int)(u % p.J);
    const lv_victim x = v[i];
    const int32_t slot = slots[i];
    if (slot < 0) continue;                          // reservation failed (error already set)
    bool ok = x.sid >= 0 && x.sid < p.S && x.blk >= 0 && x.page >= 0 && x.page < p.hbm_pages &&
              slot < p.host_pages;
    ok = ok && x.blk < nblocks_of(p, x.sid);
    ok = ok && p.table[(size_t)x.sid * p.maxB + x.blk] == x.page &&
         p.own_hbm[x.page] == owner_key(x.sid, x.blk);
    const bool clean = ok && clean_copy_of(p, x) == slot;   // its clean copy: nothing to move
    if (j == 0 && threadIdx.x == 0) {
      if (!ok) set_error(p.ctl, LV_ERR_STATE, i);
      else atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_PAGES_OUT]), 1ull);
      if (clean) atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_CLEAN_OUT]), 1ull);
      if (commit) commit[i] = lv_remap_entry{x.sid, x.blk, ok ? -(slot + 2) : -1};
    }
    if (!ok || clean) continue;
    const int4* src = reinterpret_cast<const int4*>(p.kv[j] + (size_t)x.page * p.P);
    int4* dst = reinterpret_cast<int4*>(p.host + ((size_t)slot * p.J + j) * p.P);
    copy_subpage(src, dst, nvec);
  }
}

// Unit u = (block i, sub-page j): host[slot(blk_i)][j] -> hbm_kv[j][page_i].
__global__ void __launch_bounds__(kCopyThreads)
k_swap_in(DevPool p, int32_t sid, const int32_t* __restrict__ blks,
          const int32_t* __restrict__ pages, long long n, lv_remap_entry* __restrict__ commit) {
  const long long units = n * p.J;
  const int nvec = (int)(p.P >> 4);
  const bool sid_ok = sid >= 0 && sid < p.S;
  const int32_t nb = sid_ok ? nblocks_of(p, sid) : 0;
  for (long long u = blockIdx.x; u < units; u += gridDim.x) {
    const long long i = u / p.J;
    const int j = (int)(u % p.J);
    const int32_t blk = blks[i];
    const int32_t page = pages[i];
    if (page < 0) continue;                          // reservation failed (error already set)
    bool ok = sid_ok && blk >= 0 && blk < nb && page < p.hbm_pages;
    long long slot = -1;
    if (ok) {
      const int32_t e = p.table[(size_t)sid * p.maxB + blk];
      slot = -(long long)e - 2;
      ok = e <= -2 && slot < p.host_pages && p.own_host[slot] == owner_key(sid, blk);
    }
    if (j == 0 && threadIdx.x == 0) {
      if (!ok) set_error(p.ctl, sid_ok ? LV_ERR_STATE : LV_ERR_BOUNDS, i);
      else atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_PAGES_IN]), 1ull);
      if (commit) commit[i] = lv_remap_entry{sid, blk, ok ? page : -1};
    }
    if (!ok) continue;
    const int4* src = reinterpret_cast<const int4*>(p.host + ((size_t)slot * p.J + j) * p.P);
    int4* dst = reinterpret_cast<int4*>(p.kv[j] + (size_t)page * p.P);
    copy_subpage(src, dst, nvec);
  }
}

// -------------------------------------------------------------- exchange
// Evict n_out victims and load n_in host blocks of one session in a single
// stream-ordered step whose result equals swap-out, commit, swap-in, commit
// done one after the other.  k_exchange_plan (one CTA) takes every metadata
// decision in that order -- validation, host slots (lowest free, victim
// order), out-commit, HBM pages (lowest free after the frees, list order),
// in-commit -- and emits copy tasks {out page, out slot, in slot, in page}.
// An incoming block that lands on a victim's old page shares that victim's
// task, so one thread reads the old bytes before it writes the new ones and
// both directions of the host link carry data at the same time.
constexpr int kPlanThreads = 1024;
constexpr unsigned long long kPairedBit = 1ull << 31;

// Words shared by the steps of one lv_make_resident call.
enum ResWord : int {
  R_K_SELECT = 0,   // k handed to the ranker (0 when nothing is to be evicted)
  R_N_OUT = 1,      // victims the exchange evicts
  R_N_IN = 2,       // host blocks the exchange loads
  R_STATUS = 3,     // LV_RESIDENT_*
  R_K = 4,          // pages the budget was short
  R_GATE = 5,       // 0: the append may run
  R_N_TASKS = 6,
  R_APPENDED = 7,   // int32 count of appended pages, in the low half
  R_FOUND = 8,      // victims the ranking found
  R_SID = 9,        // lv_turn: the turn's session (-1 when the pick failed)
  R_CURSOR = 10     // the exchange copy's next unit (zeroed by the plan)
};

// The gate after a device-driven step's ranking, run by the exchange plan's first
// thread before it reads the counts.  GATE_RESIDENT / GATE_PRELOAD (lv_make_resident):
// a shortfall stops the step (a preload is skipped, a foreground turn fails),
// otherwise the exchange evicts exactly k victims.  GATE_EVICT (lv_evict): every
// victim found is evicted; none found is LV_RESIDENT_NOTHING.
enum { GATE_NONE = 0, GATE_RESIDENT = 1, GATE_PRELOAD = 2, GATE_EVICT = 3 };

__device__ __forceinline__ void step_gate(const DevPool& p, long long* __restrict__ R, int gate) {
  const long long found = p.ctl[C_SEL_COUNT];   // min(k, candidates)
  if (gate == GATE_EVICT) {
    R[R_FOUND] = found;
    R[R_N_OUT] = found;
    if (found == 0) R[R_STATUS] = LV_RESIDENT_NOTHING;
    return;
  }
  if (R[R_STATUS] != LV_RESIDENT_DONE) return;
  const long long k = R[R_K];
  R[R_FOUND] = found;
  if (found < k) {
    if (gate == GATE_PRELOAD) {
      R[R_STATUS] = LV_RESIDENT_SKIPPED;
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_PRELOADS_SKIPPED]), 1ull);
    } else {
      set_error(p.ctl, LV_ERR_NO_HBM, k);
      R[R_STATUS] = LV_RESIDENT_FAILED;
    }
    R[R_N_OUT] = 0;
    R[R_N_IN] = 0;
    R[R_GATE] = 1;
  } else {
    R[R_N_OUT] = k;
  }
}

__device__ void finish_step(const DevPool& p, const StepFinish& f, const long long* __restrict__ R);

__global__ void __launch_bounds__(kPlanThreads)
k_exchange_plan(DevPool p, const lv_victim* __restrict__ v, long long n_out, int32_t sid,
                const int32_t* __restrict__ blks, long long n_in, int32_t* __restrict__ slots,
                int32_t* __restrict__ pages, int4* __restrict__ tasks, long long* n_tasks,
                int32_t epoch, unsigned long long* __restrict__ page_tag,
                const long long* counts_dev, const long long* __restrict__ sid_dev,
                long long* R, int gate, long long* __restrict__ cursor, StepFinish fin) {
  pdl_entry();
  __shared__ int bad;
  if (threadIdx.x == 0) {
    bad = 0;
    if (cursor) *cursor = 0;
    if (gate != GATE_NONE) step_gate(p, R, gate);   // a device-driven step: may set the counts
  }
  __syncthreads();
  if (counts_dev) {          // counts decided on the device (lv_make_resident, lv_evict)
    n_out = counts_dev[0];
    n_in = counts_dev[1];
  }
  if (sid_dev) sid = (int32_t)*sid_dev;
  const bool sid_ok = sid >= 0 && sid < p.S;
  const int32_t nb_in = sid_ok ? nblocks_of(p, sid) : 0;
  // validation: every victim is resident where it says, every incoming block is in
  // the host tier, and no block appears twice (victims and incoming blocks side by
  // side: item i < n_out is victim i, item n_out + i incoming block i)
  for (long long it = threadIdx.x; it < n_out + n_in; it += kPlanThreads) {
    if (it < n_out) {
      const lv_victim x = v[it];
      bool ok = x.sid >= 0 && x.sid < p.S && x.blk >= 0 && x.page >= 0 && x.page < p.hbm_pages;
      ok = ok && x.blk < nblocks_of(p, x.sid);
      ok = ok && p.table[(size_t)x.sid * p.maxB + x.blk] == x.page &&
           p.own_hbm[x.page] == owner_key(x.sid, x.blk);
      ok = ok && atomicExch(&p.mark[(size_t)x.sid * p.maxB + x.blk], epoch) != epoch;
      if (!ok) { set_error(p.ctl, LV_ERR_STATE, it); bad = 1; }
    } else {
      const int32_t b = blks[it - n_out];
      bool ok = sid_ok && b >= 0 && b < nb_in;
      if (ok) {
        const int32_t e = p.table[(size_t)sid * p.maxB + b];
        const long long h = -(long long)e - 2;
        ok = e <= -2 && h < p.host_pages && p.own_host[h] == owner_key(sid, b);
        ok = ok && atomicExch(&p.mark[(size_t)sid * p.maxB + b], epoch) != epoch;
      }
      if (!ok) { set_error(p.ctl, sid_ok ? LV_ERR_STATE : LV_ERR_BOUNDS, it); bad = 1; }
    }
  }
  __syncthreads();   // every validation verdict is in `bad` before the capacity check
  // victims without a clean copy: all of them unless the tiers are inclusive
  long long n_dirty = n_out;
  if (p.incl) {
    long long cnt = 0;
    for (long long i = threadIdx.x; i < n_out; i += kPlanThreads) cnt += clean_copy_of(p, v[i]) < 0;
    block_excl_scan<kPlanThreads>(cnt, &n_dirty);
  }
  if (threadIdx.x == 0 && !bad) {
    // capacity, as the sequential calls see it: host slots before any is freed,
    // HBM pages after the victims' pages are freed
    if (p.ctl[C_HOST_ALLOC] + n_dirty > p.host_pages) {
      set_error(p.ctl, LV_ERR_NO_HOST, n_dirty);
      bad = 1;
    } else if (p.ctl[C_HBM_ALLOC] - n_out + n_in > p.budget) {
      set_error(p.ctl, LV_ERR_NO_HBM, n_in);
      bad = 1;
    }
  }
  __syncthreads();
  if (bad) {
    for (long long i = threadIdx.x; i < n_out; i += kPlanThreads) slots[i] = -1;
    for (long long i = threadIdx.x; i < n_in; i += kPlanThreads) pages[i] = -1;
    if (threadIdx.x == 0) {
      *n_tasks = 0;
      if (fin.on) finish_step(p, fin, R);
    }
    return;
  }
  // host slots for the victims: a clean copy, or the lowest free slots in victim order
  if (n_out > 0) block_alloc_out<kPlanThreads>(p, v, n_out, n_dirty, slots);
  __syncthreads();
  // out-commit: victims now live in their slots, their pages are free; only a
  // victim that moves bytes tags its page (a clean one has nothing to read)
  const unsigned long long tag = (unsigned long long)(uint32_t)epoch << 32;
  for (long long i = threadIdx.x; i < n_out; i += kPlanThreads) {
    const lv_victim x = v[i];
    const uint32_t key = owner_key(x.sid, x.blk);
    const size_t ti = (size_t)x.sid * p.maxB + x.blk;
    const bool clean = p.incl && p.shadow[ti] == slots[i];
    p.table[ti] = -(slots[i] + 2);
    if (clean) p.shadow[ti] = -1;
    p.own_host[slots[i]] = key;
    p.own_hbm[x.page] = kOwnerNone;
    atomicAnd(&p.bits_hbm[x.page >> 5], ~(1u << (x.page & 31)));
    if (!clean) page_tag[x.page] = tag | (unsigned long long)i;
  }
  __syncthreads();
  // HBM pages for the incoming blocks
  if (n_in > 0) block_alloc_lowest<kPlanThreads>(p.bits_hbm, p.hbm_pages, n_in, pages);
  __syncthreads();
  // in-commit, and one task per incoming block (paired with the victim whose page it takes)
  for (long long i = threadIdx.x; i < n_in; i += kPlanThreads) {
    const int32_t b = blks[i];
    const size_t ti = (size_t)sid * p.maxB + b;
    const long long g = -(long long)p.table[ti] - 2;
    const int32_t pg = pages[i];
    const unsigned long long pt = page_tag[pg];   // read before this thread's stores
    p.table[ti] = pg;
    p.own_hbm[pg] = owner_key(sid, b);
    if (p.incl) {
      p.shadow[ti] = (int32_t)g;             // the host slot stays as its clean copy
    } else {
      p.own_host[g] = kOwnerNone;
      atomicAnd(&p.bits_host[g >> 5], ~(1u << (g & 31)));
    }
    int4 t = make_int4(-1, -1, (int32_t)g, pg);
    if ((pt >> 32) == (unsigned long long)(uint32_t)epoch && !(pt & kPairedBit)) {
      const long long vi = (long long)(pt & 0x7fffffffull);
      t.x = pg;
      t.y = slots[vi];
      page_tag[pg] = pt | kPairedBit;
    }
    tasks[i] = t;
  }
  __syncthreads();
  // victims whose page no incoming block takes: out-only tasks, in victim order
  long long run = 0;
  for (long long i0 = 0; i0 < n_out; i0 += kPlanThreads) {
    const long long i = i0 + threadIdx.x;
    long long flag = 0;
    int32_t pg = -1;
    if (i < n_out) {
      pg = v[i].page;
      const unsigned long long pt = page_tag[pg];
      flag = ((pt >> 32) == (unsigned long long)(uint32_t)epoch && !(pt & kPairedBit)) ? 1 : 0;
    }
    long long chunk;
    const long long pos = run + block_excl_scan<kPlanThreads>(flag, &chunk);
    if (flag) tasks[n_in + pos] = make_int4(pg, slots[i], -1, -1);
    run += chunk;
  }
  if (threadIdx.x == 0) {
    *n_tasks = n_in + run;
    const long long n_clean = n_out - n_dirty;
    const long long host_delta = p.incl ? n_dirty : n_dirty - n_in;
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_HOST_ALLOC]), (unsigned long long)host_delta);
    if (p.incl) {
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_CLEAN]), (unsigned long long)(n_in - n_clean));
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_CLEAN_OUT]), (unsigned long long)n_clean);
    }
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_HBM_ALLOC]), (unsigned long long)(n_in - n_out));
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_PAGES_OUT]), (unsigned long long)n_out);
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_PAGES_IN]), (unsigned long long)n_in);
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_REMAP]), (unsigned long long)(n_out + n_in));
    if (fin.on) finish_step(p, fin, R);   // the step's end when nothing follows the plan
  }
}

// Unit u = (task t, sub-page j): the out half copies hbm_kv[j][page] to host[slot][j],
// the in half host[slot'][j] to hbm_kv[j][page']; each thread loads both before it
// stores either, so a paired task reads the old page before overwriting it.  CTAs take
// units in order from a shared cursor (zeroed by the plan), the next one fetched while
// the current one is copied: a CTA that starts late, or runs on an SM crowded by other
// work, simply takes fewer units.
__global__ void __launch_bounds__(kCopyThreads)
k_exchange_copy(DevPool p, const int4* __restrict__ tasks, const long long* __restrict__ n_tasks,
                long long* __restrict__ cursor) {
  pdl_entry();
  const long long units = *n_tasks * p.J;
  const int nvec = (int)(p.P >> 4);
  __shared__ long long next;
  if (threadIdx.x == 0) next = (long long)atomicAdd(reinterpret_cast<unsigned long long*>(cursor), 1ull);
  __syncthreads();
  for (long long u = next; u < units; u = next) {
    // thread 0 fetches the next unit now and publishes it after the copy, so that its
    // warp does not wait for the atomic's result meanwhile
    unsigned long long fetched = 0;
    if (threadIdx.x == 0) fetched = atomicAdd(reinterpret_cast<unsigned long long*>(cursor), 1ull);
    const int4 t = tasks[u / p.J];
    const int j = (int)(u % p.J);
    const bool has_out = t.x >= 0, has_in = t.z >= 0;
    const int4* so = has_out ? reinterpret_cast<const int4*>(p.kv[j] + (size_t)t.x * p.P) : nullptr;
    int4* dout = has_out ? reinterpret_cast<int4*>(p.host + ((size_t)t.y * p.J + j) * p.P) : nullptr;
    const int4* si = has_in ? reinterpret_cast<const int4*>(p.host + ((size_t)t.z * p.J + j) * p.P) : nullptr;
    int4* din = has_in ? reinterpret_cast<int4*>(p.kv[j] + (size_t)t.w * p.P) : nullptr;
    for (int base = threadIdx.x; base < nvec; base += kCopyThreads * kCopyUnroll) {
      int4 ro[kCopyUnroll], ri[kCopyUnroll];
#pragma unroll
      for (int k = 0; k < kCopyUnroll; ++k) {
        const int q = base + k * kCopyThreads;
        if (q < nvec) {
          if (has_in) ri[k] = si[q];
          if (has_out) ro[k] = so[q];
        }
      }
#pragma unroll
      for (int k = 0; k < kCopyUnroll; ++k) {
        const int q = base + k * kCopyThreads;
        if (q < nvec) {
          if (has_out) dout[q] = ro[k];
          if (has_in) din[q] = ri[k];
        }
      }
    }
    __syncthreads();   // every thread holds u before `next` is replaced
    if (threadIdx.x == 0) next = (long long)fetched;
    __syncthreads();
  }
}

// ---------------------------------------------------------------- staged
// The staged path moves pages through a contiguous HBM staging run so that the
// copy engines can carry them over the host link: tasks (the exchange's
// {out page, out slot, in slot, in page}) are built and validated first, then
// k_pack_tasks gathers every out page's 2L sub-pages into staging[t] and
// k_unpack_tasks scatters staging[t] into every in page.  Both kernels move
// whole sub-pages with TMA bulk copies (global -> shared -> global), issued by
// one thread per CTA through a ring of shared-memory stages.

// Validated out-tasks of a swap-out: {page, slot, -1, -1} (all -1 when invalid).
__global__ void k_tasks_out(DevPool p, const lv_victim* __restrict__ v, const int32_t* __restrict__ slots,
                            long long n, int4* __restrict__ tasks, lv_remap_entry* __restrict__ commit) {
  const long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  if (i >= n) return;
  const lv_victim x = v[i];
  const int32_t slot = slots[i];
  int4 t = make_int4(-1, -1, -1, -1);
  if (slot >= 0) {
    bool ok = x.sid >= 0 && x.sid < p.S && x.blk >= 0 && x.page >= 0 && x.page < p.hbm_pages &&
              slot < p.host_pages;
    ok = ok && x.blk < nblocks_of(p, x.sid);
    ok = ok && p.table[(size_t)x.sid * p.maxB + x.blk] == x.page &&
         p.own_hbm[x.page] == owner_key(x.sid, x.blk);
    if (!ok) set_error(p.ctl, LV_ERR_STATE, i);
    else {
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_PAGES_OUT]), 1ull);
      if (clean_copy_of(p, x) == slot)        // its clean copy: no task
        atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_CLEAN_OUT]), 1ull);
      else
        t = make_int4(x.page, slot, -1, -1);
    }
    if (commit) commit[i] = lv_remap_entry{x.sid, x.blk, ok ? -(slot + 2) : -1};
  } else if (commit) {
    commit[i] = lv_remap_entry{x.sid, x.blk, -1};
  }
  tasks[i] = t;
}

// Validated in-tasks of a swap-in: {-1, -1, slot, page} (all -1 when invalid).
__global__ void k_tasks_in(DevPool p, int32_t sid, const int32_t* __restrict__ blks,
                           const int32_t* __restrict__ pages, long long n, int4* __restrict__ tasks,
                           lv_remap_entry* __restrict__ commit) {
  const long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  if (i >= n) return;
  const int32_t blk = blks[i], page = pages[i];
  int4 t = make_int4(-1, -1, -1, -1);
  const bool sid_ok = sid >= 0 && sid < p.S;
  if (page >= 0) {
    bool ok = sid_ok && blk >= 0 && blk < nblocks_of(p, sid) && page < p.hbm_pages;
    long long slot = -1;
    if (ok) {
      const int32_t e = p.table[(size_t)sid * p.maxB + blk];
      slot = -(long long)e - 2;
      ok = e <= -2 && slot < p.host_pages && p.own_host[slot] == owner_key(sid, blk);
    }
    if (!ok) set_error(p.ctl, sid_ok ? LV_ERR_STATE : LV_ERR_BOUNDS, i);
    else {
      t = make_int4(-1, -1, (int32_t)slot, page);
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_PAGES_IN]), 1ull);
    }
    if (commit) commit[i] = lv_remap_entry{sid, blk, ok ? page : -1};
  } else if (commit) {
    commit[i] = lv_remap_entry{sid, blk, -1};
  }
  tasks[i] = t;
}

__device__ __forceinline__ uint32_t smem_addr(const void* ptr) {
  return (uint32_t)__cvta_generic_to_shared(ptr);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return done != 0;
}

// 1-D bulk copy global -> this CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_load(void* dst_smem, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst_smem)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

// 1-D bulk copy shared -> global, tracked by the bulk async-group.
__device__ __forceinline__ void bulk_store(void* dst, const void* src_smem, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst),
               "r"(smem_addr(src_smem)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_all() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_read_1() {
  asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded wait on a stage barrier: false once `limit_ns` have passed (the data never came).
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, long long limit_ns) {
  const unsigned long long t0 = global_ns();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((long long)(global_ns() - t0) > limit_ns) return false;
  }
}

constexpr int kStageThreads = 32;     // one warp per CTA; lane 0 issues the bulk copies
constexpr int kMaxStages = 16;
constexpr long long kWaitLimitNs = 1000000000ll;   // one second per stage wait

// Moves units u = (task t, sub-page j) of P bytes through `stages` shared-memory
// buffers: unit i's load is issued `stages` units ahead of its store.
// pack:   staging[t][j] <- hbm_kv[j][task.x]   for tasks with task.x >= 0
// unpack: hbm_kv[j][task.w] <- staging[t][j]   for tasks with task.z >= 0
template <bool kPack>
__global__ void __launch_bounds__(kStageThreads)
k_stage_tasks(DevPool p, const int4* __restrict__ tasks, long long t_begin, long long t_end,
              uint8_t* __restrict__ staging, int stages) {
  extern __shared__ __align__(128) unsigned char stage_mem[];
  __shared__ __align__(8) uint64_t bars[kMaxStages];
  if (threadIdx.x != 0) return;
  const uint32_t P = (uint32_t)p.P;
  for (int s = 0; s < stages; ++s) mbar_init(&bars[s], 1);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  const long long units = (t_end - t_begin) * p.J;
  // the units of this CTA, in order: u = blockIdx.x + k * gridDim.x
  auto unit_ptrs = [&](long long k, const uint8_t** src, uint8_t** dst) -> bool {
    const long long u = blockIdx.x + k * (long long)gridDim.x;
    const long long t = t_begin + u / p.J;
    const int j = (int)(u % p.J);
    const int4 tk = tasks[t];
    uint8_t* st = staging + ((size_t)t * p.J + j) * P;
    if (kPack) {
      if (tk.x < 0) return false;
      *src = p.kv[j] + (size_t)tk.x * P;
      *dst = st;
    } else {
      if (tk.z < 0) return false;
      *src = st;
      *dst = p.kv[j] + (size_t)tk.w * P;
    }
    return true;
  };
  const long long mine = units > blockIdx.x ? (units - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
  uint8_t* dsts[kMaxStages];
  bool live[kMaxStages];
  uint32_t phase[kMaxStages];
  for (int s = 0; s < stages; ++s) { live[s] = false; phase[s] = 0; }
  bool failed = false;
  auto issue = [&](long long k) {
    const int s = (int)(k % stages);
    const uint8_t* src;
    live[s] = unit_ptrs(k, &src, &dsts[s]);
    if (live[s]) {
      mbar_expect_tx(&bars[s], P);
      bulk_load(stage_mem + (size_t)s * P, src, P, &bars[s]);
    }
  };
  // prologue: one load in flight per stage
  for (long long k = 0; k < mine && k < stages; ++k) issue(k);
  for (long long k = 0; k < mine; ++k) {
    const int s = (int)(k % stages);
    bool stored = false;
    if (live[s]) {
      if (!mbar_wait_bounded(&bars[s], phase[s], kWaitLimitNs)) {
        failed = true;
        break;
      }
      phase[s] ^= 1u;
      bulk_store(dsts[s], stage_mem + (size_t)s * P, P);
      bulk_commit();
      stored = true;
    }
    // refill the stage of unit k-1 once its store has read it; unit k's store may still run
    if (k >= 1 && k - 1 + stages < mine) {
      if (stored) bulk_wait_read_1();
      else bulk_wait_read_all();
      issue(k - 1 + stages);
    }
  }
  if (failed) {
    set_error(p.ctl, LV_ERR_TIMEOUT, blockIdx.x);
    // let every load still in flight land before the shared memory is released
    for (int s = 0; s < stages; ++s)
      if (live[s]) mbar_wait_bounded(&bars[s], phase[s], kWaitLimitNs);
  }
  bulk_wait_all();
}

// The exchange's copies with TMA bulk copies instead of the SMs' loads and stores:
// one thread per CTA moves units u = (task, sub-page j) through `stages`
// shared-memory stages of 2P bytes.  A unit's out half (old HBM page -> its new host
// slot) and in half (host slot -> its new HBM page) are loaded into one stage
// together and stored from it once both have arrived, so a paired task's page is
// read before it is overwritten.  Units come from the shared cursor (zeroed by the
// plan) kXBatch at a time; a CTA refills the stage of unit k-1 while unit k's stores
// still run.  The CTA issues a few instructions per 2P bytes, so its SM stays free
// for other work; every barrier wait is bounded (LV_ERR_TIMEOUT).
constexpr int kXStageMax = 8;
constexpr int kXBatch = 8;

__global__ void __launch_bounds__(kStageThreads)
k_exchange_copy_tma(DevPool p, const int4* __restrict__ tasks, const long long* __restrict__ n_tasks,
                    long long* __restrict__ cursor) {
  extern __shared__ __align__(128) unsigned char xmem[];
  __shared__ __align__(8) uint64_t bars[kXStageMax];
  pdl_entry();
  if (threadIdx.x != 0) return;
  const int stages = p.xstages;
  const uint32_t P = (uint32_t)p.P;
  const long long units = *n_tasks * p.J;
  for (int s = 0; s < stages; ++s) mbar_init(&bars[s], 1);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  uint8_t* dout[kXStageMax];
  uint8_t* din[kXStageMax];
  bool pending[kXStageMax];
  uint32_t phase[kXStageMax];
  for (int s = 0; s < stages; ++s) {
    dout[s] = din[s] = nullptr;
    pending[s] = false;
    phase[s] = 0;
  }
  long long ub = 0, ue = 0, taken = 0;
  bool exhausted = false;
  // takes the CTA's unit number k (its k-th, in order) into stage k % stages
  auto take = [&](long long k) {
    if (exhausted) return;
    if (ub == ue) {
      ub = (long long)atomicAdd(reinterpret_cast<unsigned long long*>(cursor), (unsigned long long)kXBatch);
      ue = ub + kXBatch < units ? ub + kXBatch : units;
      if (ub >= units) {
        exhausted = true;
        return;
      }
    }
    const long long u = ub++;
    const int s = (int)(k % stages);
    const int4 t = tasks[u / p.J];
    const int j = (int)(u % p.J);
    unsigned char* so = xmem + (size_t)s * 2 * P;
    dout[s] = t.x >= 0 ? p.host + ((size_t)t.y * p.J + j) * P : nullptr;
    din[s] = t.z >= 0 ? p.kv[j] + (size_t)t.w * P : nullptr;
    const uint32_t bytes = (t.x >= 0 ? P : 0u) + (t.z >= 0 ? P : 0u);
    pending[s] = bytes > 0;
    if (bytes) {
      mbar_expect_tx(&bars[s], bytes);
      if (t.x >= 0) bulk_load(so, p.kv[j] + (size_t)t.x * P, P, &bars[s]);
      if (t.z >= 0) bulk_load(so + P, p.host + ((size_t)t.z * p.J + j) * P, P, &bars[s]);
    }
    taken = k + 1;
  };
  for (long long k = 0; k < stages; ++k) take(k);
  bool failed = false;
  for (long long k = 0; k < taken; ++k) {
    const int s = (int)(k % stages);
    bool stored = false;
    if (pending[s]) {
      if (!mbar_wait_bounded(&bars[s], phase[s], kWaitLimitNs)) {
        failed = true;
        break;
      }
      pending[s] = false;
      phase[s] ^= 1u;
      unsigned char* so = xmem + (size_t)s * 2 * P;
      if (dout[s]) bulk_store(dout[s], so, P);
      if (din[s]) bulk_store(din[s], so + P, P);
      bulk_commit();
      stored = true;
    }
    // refill the stage of unit k-1 once its stores have read it; unit k's may still run
    if (k >= 1 && !exhausted) {
      if (stored) bulk_wait_read_1();
      else bulk_wait_read_all();
      take(k - 1 + stages);
    }
  }
  if (failed) {
    set_error(p.ctl, LV_ERR_TIMEOUT, blockIdx.x);
    // let every load still in flight land before the shared memory is released
    for (int s = 0; s < stages; ++s)
      if (pending[s]) mbar_wait_bounded(&bars[s], phase[s], kWaitLimitNs);
  }
  bulk_wait_all();
}

// The same moves with plain 16-byte loads and stores (256 threads per CTA).
template <bool kPack>
__global__ void __launch_bounds__(kCopyThreads)
k_stage_tasks_lsu(DevPool p, const int4* __restrict__ tasks, long long t_begin, long long t_end,
                  uint8_t* __restrict__ staging) {
  const long long units = (t_end - t_begin) * p.J;
  const int nvec = (int)(p.P >> 4);
  for (long long u = blockIdx.x; u < units; u += gridDim.x) {
    const long long t = t_begin + u / p.J;
    const int j = (int)(u % p.J);
    const int4 tk = tasks[t];
    uint8_t* st = staging + ((size_t)t * p.J + j) * p.P;
    if (kPack) {
      if (tk.x < 0) continue;
      copy_subpage(reinterpret_cast<const int4*>(p.kv[j] + (size_t)tk.x * p.P), reinterpret_cast<int4*>(st), nvec);
    } else {
      if (tk.z < 0) continue;
      copy_subpage(reinterpret_cast<const int4*>(st), reinterpret_cast<int4*>(p.kv[j] + (size_t)tk.w * p.P), nvec);
    }
  }
}

// Tasks for a plain list of pages: pack reads them ({page, -1, -1, -1}), unpack
// writes them ({-1, -1, 0, page}); an out-of-range page gives an empty task.
__global__ void k_tasks_pages(DevPool p, const int32_t* __restrict__ pages, long long n, bool pack,
                              int4* __restrict__ tasks) {
  const long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  if (i >= n) return;
  const int32_t pg = pages[i];
  if (pg < 0 || pg >= p.hbm_pages) {
    set_error(p.ctl, LV_ERR_BOUNDS, i);
    tasks[i] = make_int4(-1, -1, -1, -1);
    return;
  }
  tasks[i] = pack ? make_int4(pg, -1, -1, -1) : make_int4(-1, -1, 0, pg);
}

// Self-test of the bounded wait: one thread arms a stage barrier for bytes that no
// copy will ever deliver and waits on it with the given limit; the timeout must be
// reported in the error word and the kernel must return.
__global__ void k_selftest_wait(long long* ctl, long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  mbar_expect_tx(&bar, 16);                       // 16 bytes that never arrive
  if (!mbar_wait_bounded(&bar, 0, limit_ns)) set_error(ctl, LV_ERR_TIMEOUT, limit_ns);
}

// ---------------------------------------------------------------- commit
constexpr int kRemapThreads = 256;
constexpr int kReleaseThreads = 256;

// The reads of one entry that do not depend on a check.
struct RemapRead {
  lv_remap_entry x;
  size_t ti;            // table index (0 when out of range)
  int32_t old;          // the block's current location
  int32_t g;            // its clean-copy slot (inclusive tiers), or -1
  int32_t nb;           // blocks of its session
  bool in_range;
};

struct RemapCounts {
  int ok, hbm, host, clean;
};

__device__ __forceinline__ void remap_read_entry(const DevPool& p, const lv_remap_entry* e, long long i,
                                                 long long n, RemapRead& r) {
  r.x = i < n ? e[i] : lv_remap_entry{-1, -1, -1};
  r.in_range = i < n && r.x.sid >= 0 && r.x.sid < p.S && r.x.blk >= 0 && r.x.blk < p.maxB;
  r.ti = r.in_range ? (size_t)r.x.sid * p.maxB + r.x.blk : 0;
}

__device__ __forceinline__ void remap_read_table(const DevPool& p, RemapRead& r) {
  r.old = r.in_range ? p.table[r.ti] : -1;
  r.g = (r.in_range && p.incl) ? p.shadow[r.ti] : -1;
  r.nb = r.in_range ? nblocks_of(p, r.x.sid) : 0;
}

// The block's epoch mark: one accepted entry per block per call.  It depends on
// the entry alone, so it is issued with the entry's table reads; a mark made for
// a block past its session's context is harmless (every entry naming that block
// fails the same range check).  A returning atomic: the caller issues every
// entry's mark before it looks at any result.
__device__ __forceinline__ void remap_mark(const DevPool& p, const RemapRead& r, int32_t epoch,
                                           int32_t& seen) {
  seen = r.in_range ? atomicExch(&p.mark[r.ti], epoch) : 0;
}

// The entry's error once its table reads and mark are back: range first, then
// a second entry for the same block.
__device__ __forceinline__ int remap_judge(const RemapRead& r, int32_t epoch, int32_t seen) {
  if (!r.in_range || r.x.blk >= r.nb) return LV_ERR_BOUNDS;
  if (seen == epoch) return LV_ERR_DOUBLE_MAP;
  return 0;
}

// Round 3 of an entry that passed its range check and its mark.  The claim of the
// new location (one CAS checks that it is a reservation nobody owns and takes it)
// goes out together with the entry's own writes, made before the claim's result
// is known: the table word, and the old location exchanged to kOwnerFreeing
// (which returns its owner word into `was`, for the consistency check).  The
// release pass after the commit makes a kOwnerFreeing word free and clears its
// bitmap bit.  A claim that fails undoes the writes in remap_settle; until then
// no other entry of the call can see them, since only an entry for the same
// block reads its table word (and the mark turned it away), and every claim of
// an owned location fails, kOwnerFreeing or not.
__device__ __forceinline__ int remap_claim(const DevPool& p, const RemapRead& r, int err,
                                           uint32_t& got, uint32_t& was) {
  if (err) return err;
  const lv_remap_entry& x = r.x;
  const uint32_t key = owner_key(x.sid, x.blk);
  uint32_t* own;
  if (x.loc >= 0) {
    if (x.loc >= p.hbm_pages) return LV_ERR_BOUNDS;
    own = &p.own_hbm[x.loc];
  } else if (x.loc <= -2) {
    if (-(long long)x.loc - 2 >= p.host_pages) return LV_ERR_BOUNDS;
    own = &p.own_host[-(long long)x.loc - 2];
  } else {
    return LV_ERR_BOUNDS;
  }
  got = atomicCAS(own, kOwnerReserved, key);
  const int32_t old = r.old;
  const long long old_slot = -(long long)old - 2;
  if (old >= 0 && old < p.hbm_pages) {
    was = atomicExch(&p.own_hbm[old], kOwnerFreeing);
  } else if (old <= -2 && old_slot < p.host_pages) {
    if (p.incl && x.loc >= 0) was = p.own_host[old_slot];   // back in HBM: the slot stays as its clean copy
    else was = atomicExch(&p.own_host[old_slot], kOwnerFreeing);
  }
  p.table[r.ti] = x.loc;
  return 0;
}

// Judges the claim once its result is back.  A failed claim is a double map and
// its entry's writes are put back; an accepted entry settles its clean copy
// (inclusive tiers) and is counted, and a freed location that this block did not
// own means the tables were inconsistent.
__device__ __forceinline__ void remap_settle(const DevPool& p, const RemapRead& r, int err,
                                             uint32_t got, uint32_t was, long long i,
                                             RemapCounts& c) {
  const lv_remap_entry& x = r.x;
  const int32_t old = r.old, g = r.g;
  const long long old_slot = -(long long)old - 2;
  const bool old_hbm = old >= 0 && old < p.hbm_pages;
  const bool old_host = old <= -2 && old_slot < p.host_pages;
  const long long h = -(long long)x.loc - 2;
  const uint32_t key = owner_key(x.sid, x.blk);
  if (!err && got != kOwnerReserved) {
    // a host location already owned by this block is fine only as its own clean copy
    if (!(x.loc <= -2 && p.incl && (long long)g == h && got == key)) {
      err = LV_ERR_DOUBLE_MAP;
      p.table[r.ti] = old;
      if (old_hbm) p.own_hbm[old] = was;
      else if (old_host && !(p.incl && x.loc >= 0)) p.own_host[old_slot] = was;
    }
  }
  if (err) {
    set_error(p.ctl, err, i);
    return;
  }
  if (x.loc <= -2 && g >= 0) {          // the copy becomes the location, or goes
    p.shadow[r.ti] = -1;
    c.clean -= 1;
    if ((long long)g != h) {
      atomicExch(&p.own_host[g], kOwnerFreeing);
      c.host += 1;
    }
  }
  if (old_hbm) {
    c.hbm += 1;
  } else if (old_host) {
    if (p.incl && x.loc >= 0) {
      p.shadow[r.ti] = (int32_t)old_slot;
      c.clean += 1;
    } else {
      c.host += 1;
    }
  }
  if (was != kOwnerNone && was != key) set_error(p.ctl, LV_ERR_STATE, i);
  c.ok += 1;
}

// Each thread commits E entries, i0, i0 + stride, ... (stride = the grid's
// threads, so a warp's entries stay contiguous).  The allocation counts and the
// commit counter change by block totals (one atomic per block and counter).
// Inclusive tiers: a host location may be the block's own clean copy; a block
// committed to HBM from the host tier keeps its slot as its clean copy; a
// block committed to another host slot loses its copy.
//
// The kernel is bound by the latency of dependent scattered accesses, so each
// round of requests is issued for all E entries of the thread before any of its
// results is used, and requests that do not depend on one another share a
// round: (1) the entries; (2) the block's table word, its session's block count
// and the block's epoch mark; (3) the claim of the new location, the table word
// and the exchange of the old location's owner word (only for an entry that
// passed its range check and its mark; the writes are undone if the claim
// fails).  E chains then wait together.  The early reads are race-free within
// one call: a block has at most one accepted entry (the epoch mark), a location
// freed by one entry is never the new location of another (new locations are
// reservations), and another entry can take an owned location only through a
// CAS, which then fails.  A thread's own entries are issued in order, so a
// duplicate among them meets the epoch mark too.
template <int E>
__global__ void __launch_bounds__(kRemapThreads, 4)
k_remap(DevPool p, const lv_remap_entry* __restrict__ e, long long n, int32_t epoch) {
  const long long stride = (long long)gridDim.x * kRemapThreads;
  const long long i0 = blockIdx.x * (long long)kRemapThreads + threadIdx.x;
  RemapRead r[E];
  int32_t seen[E];
#pragma unroll
  for (int j = 0; j < E; ++j) remap_read_entry(p, e, i0 + j * stride, n, r[j]);
#pragma unroll
  for (int j = 0; j < E; ++j) {
    remap_read_table(p, r[j]);
    remap_mark(p, r[j], epoch, seen[j]);
  }
  int err[E];
  uint32_t got[E], was[E];
#pragma unroll
  for (int j = 0; j < E; ++j) {
    got[j] = kOwnerReserved;
    was[j] = kOwnerNone;
    err[j] = i0 + j * stride < n ? remap_judge(r[j], epoch, seen[j]) : -1;
    if (err[j] >= 0) err[j] = remap_claim(p, r[j], err[j], got[j], was[j]);
  }
  RemapCounts c{0, 0, 0, 0};
#pragma unroll
  for (int j = 0; j < E; ++j)
    if (err[j] >= 0) remap_settle(p, r[j], err[j], got[j], was[j], i0 + j * stride, c);
  // block totals: warp sums, one shared atomic per warp, one global atomic per block
  __shared__ int tot[4];
  if (threadIdx.x < 4) tot[threadIdx.x] = 0;
  __syncthreads();
  const int ok = __reduce_add_sync(0xffffffffu, c.ok), fh = __reduce_add_sync(0xffffffffu, c.hbm);
  const int fo = __reduce_add_sync(0xffffffffu, c.host), cl = __reduce_add_sync(0xffffffffu, c.clean);
  if ((threadIdx.x & 31) == 0) {
    if (ok) atomicAdd(&tot[0], ok);
    if (fh) atomicAdd(&tot[1], fh);
    if (fo) atomicAdd(&tot[2], fo);
    if (cl) atomicAdd(&tot[3], cl);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (tot[1]) atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_HBM_ALLOC]), (unsigned long long)-(long long)tot[1]);
    if (tot[2]) atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_HOST_ALLOC]), (unsigned long long)-(long long)tot[2]);
    if (tot[0]) atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_REMAP]), (unsigned long long)tot[0]);
    if (tot[3]) atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_CLEAN]), (unsigned long long)(long long)tot[3]);
  }
}

// The commit's second pass: every owner word that the commit exchanged to
// kOwnerFreeing becomes kOwnerNone, and its bit is cleared in the allocation
// bitmap with one reduction per bitmap word (the commit itself would issue one
// reduction per freed page, 32 to a word when a whole run of pages is freed).
// Thread q reads owner words 4q..4q+3 of its tier with one 16-byte load; the 8
// threads of a bitmap word combine their bits with shuffles.  Quads [0, qh) are
// the HBM pages and [qh, qh + qo) the host slots; qh and qo are multiples of 8,
// so the 8 threads of a word are always 8 aligned lanes of one tier.  Each thread
// issues the loads of kReleaseUnroll quads, a grid's width apart, before it looks
// at any of them.  Only the freed words are written, so concurrent work on other
// pages is left alone.
constexpr int kReleaseUnroll = 2;

__device__ __forceinline__ uint4 release_load(const DevPool& p, long long q, long long qh,
                                              long long total) {
  uint4 v = make_uint4(kOwnerNone, kOwnerNone, kOwnerNone, kOwnerNone);
  if (q >= total) return v;
  const bool hbm = q < qh;
  const uint32_t* own = hbm ? p.own_hbm : p.own_host;
  const long long n = hbm ? p.hbm_pages : p.host_pages;
  const long long base = (hbm ? q : q - qh) * 4;
  if (base + 3 < n) {
    v = *reinterpret_cast<const uint4*>(own + base);
  } else {
    if (base < n) v.x = own[base];
    if (base + 1 < n) v.y = own[base + 1];
    if (base + 2 < n) v.z = own[base + 2];
  }
  return v;
}

__device__ __forceinline__ void release_apply(const DevPool& p, long long q, long long qh,
                                              long long total, uint4 v, int lane8) {
  const bool hbm = q < qh;
  uint32_t* own = hbm ? p.own_hbm : p.own_host;
  const long long base = (hbm ? q : q - qh) * 4;
  uint32_t m = 0;
  if (q < total) {
    m = (uint32_t)(v.x == kOwnerFreeing) | (uint32_t)(v.y == kOwnerFreeing) << 1 |
        (uint32_t)(v.z == kOwnerFreeing) << 2 | (uint32_t)(v.w == kOwnerFreeing) << 3;
    for (int k = 0; k < 4; ++k)
      if (m >> k & 1u) own[base + k] = kOwnerNone;
  }
  uint32_t w = m << (4 * lane8);
  w |= __shfl_xor_sync(0xffffffffu, w, 1);
  w |= __shfl_xor_sync(0xffffffffu, w, 2);
  w |= __shfl_xor_sync(0xffffffffu, w, 4);
  if (lane8 == 0 && w) atomicAnd(&(hbm ? p.bits_hbm : p.bits_host)[base >> 5], ~w);
}

__global__ void __launch_bounds__(kReleaseThreads)
k_release(DevPool p, long long qh, long long qo) {
  pdl_wait();   // the commit is complete and visible
  const long long total = qh + qo;
  const long long step = (long long)gridDim.x * kReleaseThreads;
  const int lane8 = threadIdx.x & 7;
  for (long long q0 = (long long)blockIdx.x * kReleaseThreads + threadIdx.x;
       q0 - threadIdx.x < total; q0 += kReleaseUnroll * step) {
    uint4 v[kReleaseUnroll];
#pragma unroll
    for (int u = 0; u < kReleaseUnroll; ++u) v[u] = release_load(p, q0 + u * step, qh, total);
#pragma unroll
    for (int u = 0; u < kReleaseUnroll; ++u) release_apply(p, q0 + u * step, qh, total, v[u], lane8);
  }
}

__global__ void k_cancel(DevPool p, const int32_t* __restrict__ locs, long long n) {
  const long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  if (i >= n) return;
  const int32_t loc = locs[i];
  uint32_t* bits;
  uint32_t* own;
  long long idx;
  int which;
  if (loc >= 0 && loc < p.hbm_pages) {
    bits = p.bits_hbm; own = p.own_hbm; idx = loc; which = C_HBM_ALLOC;
  } else if (loc <= -2 && (-(long long)loc - 2) < p.host_pages) {
    bits = p.bits_host; own = p.own_host; idx = -(long long)loc - 2; which = C_HOST_ALLOC;
  } else {
    set_error(p.ctl, LV_ERR_BOUNDS, i);
    return;
  }
  // only a pending reservation can be released; a clean copy was never reserved
  const uint32_t o = atomicCAS(&own[idx], kOwnerReserved, kOwnerNone);
  if (o != kOwnerReserved) {
    const int32_t os = (int32_t)(o >> 16), ob = (int32_t)(o & 0xFFFFu);
    const bool copy = p.incl && which == C_HOST_ALLOC && o != kOwnerNone && os < p.S &&
                      ob < p.maxB && p.shadow[(size_t)os * p.maxB + ob] == idx;
    if (!copy) set_error(p.ctl, LV_ERR_STATE, i);
    return;
  }
  const uint32_t m = 1u << (idx & 31);
  atomicAnd(&bits[idx >> 5], ~m);
  atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[which]), (unsigned long long)-1ll);
  atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_CANCELS]), 1ull);
}

__global__ void __launch_bounds__(kAllocThreads)
k_append(DevPool p, int32_t sid, int32_t n_tokens, int32_t* __restrict__ pages,
         int32_t* __restrict__ count, const long long* __restrict__ gate,
         const long long* __restrict__ sid_dev, StepFinish fin, const long long* __restrict__ R) {
  pdl_entry();
  __shared__ long long m_s, nb_s, ctx_s;
  if (gate && *gate != 0) {   // an earlier step of lv_make_resident did not complete
    if (threadIdx.x == 0) {
      if (count) *count = 0;
      if (fin.on) finish_step(p, fin, R);
    }
    return;
  }
  if (sid_dev) sid = (int32_t)*sid_dev;
  if (threadIdx.x == 0) {
    long long m = -1;
    if (sid >= 0 && sid < p.S && n_tokens >= 0) {
      const long long ctx = p.sess[sid].ctx_tokens;
      const long long nb = (ctx + p.T - 1) / p.T;
      const long long nctx = ctx + n_tokens;
      const long long nnb = (nctx + p.T - 1) / p.T;
      if (nnb > p.maxB || nctx > 0x7fffffffll) {
        set_error(p.ctl, LV_ERR_BOUNDS, sid);
      } else {
        m = nnb - nb;
        if (m > 0) {
          const long long before = (long long)atomicAdd(
              reinterpret_cast<unsigned long long*>(&p.ctl[C_HBM_ALLOC]), (unsigned long long)m);
          if (before + m > p.budget) {
            atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_HBM_ALLOC]),
                      (unsigned long long)(-m));
            set_error(p.ctl, LV_ERR_NO_HBM, sid);
            m = -1;
          }
        }
      }
      nb_s = nb;
      ctx_s = nctx;
    } else {
      set_error(p.ctl, LV_ERR_BOUNDS, sid);
    }
    m_s = m;
  }
  __syncthreads();
  const long long m = m_s;
  if (m < 0) {
    if (threadIdx.x == 0) {
      if (count) *count = 0;
      if (fin.on) finish_step(p, fin, R);
    }
    return;
  }
  if (m > 0) block_alloc_lowest<kAllocThreads>(p.bits_hbm, p.hbm_pages, m, pages);
  __syncthreads();
  for (long long i = threadIdx.x; i < m; i += kAllocThreads) {
    const int32_t pg = pages[i];
    const int32_t b = (int32_t)(nb_s + i);
    p.table[(size_t)sid * p.maxB + b] = pg;
    p.own_hbm[pg] = owner_key(sid, b);
  }
  if (threadIdx.x == 0) {
    // inclusive tiers: the partially filled last block gains rows, its clean copy is stale
    const long long old_ctx = ctx_s - n_tokens;
    if (p.incl && n_tokens > 0 && nb_s > 0 && old_ctx % p.T != 0) {
      const size_t ti = (size_t)sid * p.maxB + (nb_s - 1);
      const int32_t g = p.shadow[ti];
      if (g >= 0 && g < p.host_pages) {
        p.shadow[ti] = -1;
        p.own_host[g] = kOwnerNone;
        atomicAnd(&p.bits_host[g >> 5], ~(1u << (g & 31)));
        atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_HOST_ALLOC]), (unsigned long long)-1ll);
        atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_CLEAN]), (unsigned long long)-1ll);
        atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_CLEAN_DROPPED]), 1ull);
      }
    }
    p.sess[sid].ctx_tokens = (int32_t)ctx_s;
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_APPENDED]), (unsigned long long)m);
    if (count) *count = (int32_t)m;
    if (fin.on) finish_step(p, fin, R);   // a device-driven step's end, after its growth
  }
}

// -------------------------------------------------------- make_resident

// lv_turn's start, run first by k_resident_prepare: the turn's session (sid, or the
// first candidate with a hit, else the first candidate) into R[R_SID], then
// LV_EV_TURN_BEGIN for it.  Returns the session, -1 when the pick failed.
__device__ int32_t turn_begin(const DevPool& p, int32_t sid, const TurnStart& ts, long long* R) {
  __shared__ int first;
  __shared__ int32_t picked;
  if (threadIdx.x == 0) first = ts.n_cand;
  __syncthreads();
  if (sid < 0) {
    int mine = ts.n_cand;
    for (int c = threadIdx.x; c < ts.n_cand; c += blockDim.x)
      if (ts.hit[c]) { mine = c; break; }
    if (mine < ts.n_cand) atomicMin(&first, mine);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int32_t s = sid;
    if (s < 0) {
      const int c = first < ts.n_cand ? first : 0;
      s = ts.cand[c];
      if (s < 0 || s >= p.S) {
        set_error(p.ctl, LV_ERR_BOUNDS, c);
        s = -1;
      }
    }
    R[R_SID] = s;
    if (s >= 0) {
      lv_session_state st = p.sess[s];
      lv_event x{};
      x.kind = LV_EV_TURN_BEGIN;
      x.sid = s;
      x.t_us = ts.now_us;
      apply_event(p, st, x);
      p.sess[s] = st;
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_EVENTS]), 1ull);
    }
    picked = s;
  }
  __syncthreads();
  return picked;
}

// One CTA: sid's host-tier blocks (ascending), the deficit k and the admission; for
// lv_turn (ts.on) the turn's start first.
__global__ void __launch_bounds__(kCensusThreads)
k_resident_prepare(DevPool p, int32_t sid, int32_t append_tokens, bool preload,
                   long long max_load, int32_t* __restrict__ blocks, long long* __restrict__ R,
                   const long long* __restrict__ sid_dev, TurnStart ts) {
  pdl_entry();
  if (ts.on) sid = turn_begin(p, sid, ts, R);
  else if (sid_dev) sid = (int32_t)*sid_dev;
  if (sid < 0 || sid >= p.S) {        // lv_turn's pick failed (already reported)
    if (threadIdx.x == 0) {
      R[R_K_SELECT] = 0; R[R_N_OUT] = 0; R[R_N_IN] = 0; R[R_STATUS] = LV_RESIDENT_FAILED;
      R[R_K] = 0; R[R_GATE] = 1; R[R_APPENDED] = 0; R[R_FOUND] = 0;
    }
    return;
  }
  const int32_t nb = nblocks_of(p, sid);
  const int32_t* row = p.table + (size_t)sid * p.maxB;
  long long run = 0;
  for (int32_t q0 = 0; q0 < nb; q0 += kCensusThreads) {
    const int32_t b = q0 + threadIdx.x;
    const long long flag = (b < nb && row[b] <= -2) ? 1 : 0;
    long long chunk;
    const long long pos = run + block_excl_scan<kCensusThreads>(flag, &chunk);
    if (flag) blocks[pos] = b;
    run += chunk;
  }
  if (threadIdx.x == 0) {
    const long long nh = run;
    const long long ctx = p.sess[sid].ctx_tokens;
    const long long nctx = ctx + append_tokens;
    const long long nnb = (nctx + p.T - 1) / p.T;
    int status = LV_RESIDENT_DONE;
    long long k = 0;
    if (nnb > p.maxB || nctx > 0x7fffffffll) {
      set_error(p.ctl, LV_ERR_BOUNDS, sid);
      status = LV_RESIDENT_FAILED;
    } else {
      const long long need = nh + (nnb - nb);
      const long long free_pages = p.budget - p.ctl[C_HBM_ALLOC];
      k = need - free_pages > 0 ? need - free_pages : 0;
      if (preload && nh == 0) status = LV_RESIDENT_NOTHING;
      else if (preload && max_load >= 0 && nh > max_load) status = LV_RESIDENT_SKIPPED;
    }
    const bool go = status == LV_RESIDENT_DONE;
    R[R_K_SELECT] = go ? k : 0;
    R[R_N_OUT] = 0;
    R[R_N_IN] = go ? nh : 0;
    R[R_STATUS] = status;
    R[R_K] = k;
    R[R_GATE] = go ? 0 : 1;
    R[R_APPENDED] = 0;
    R[R_FOUND] = 0;
    if (preload && status == LV_RESIDENT_SKIPPED)
      atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_PRELOADS_SKIPPED]), 1ull);
  }
}

constexpr int kOrderThreads = 256;

// The caller's load order: host-tier block i of the session (ascending in
// `blocks`, R[R_N_IN] of them) goes to position #{j : (key[b_j], b_j) <
// (key[b_i], b_i)} of `loads` -- ascending (key, block id).  One warp per block.
__global__ void __launch_bounds__(kOrderThreads)
k_order_loads(const long long* __restrict__ R, const int32_t* __restrict__ blocks,
              const unsigned long long* __restrict__ key, int32_t* __restrict__ loads) {
  pdl_entry();
  const long long nh = R[R_N_IN];
  const long long i = blockIdx.x * (long long)(kOrderThreads / 32) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (i >= nh) return;
  const int32_t bi = blocks[i];
  const unsigned long long ki = key[bi];
  int rank = 0;
  for (long long j = lane; j < nh; j += 32) {
    const int32_t bj = blocks[j];
    const unsigned long long kj = key[bj];
    rank += (kj < ki || (kj == ki && bj < bi)) ? 1 : 0;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) rank += __shfl_xor_sync(0xffffffffu, rank, o);
  if (lane == 0) loads[rank] = bi;
}


// The step's result and, for lv_turn (turn_end), LV_EV_TURN_END for the turn's session
// unless its KV could not be made resident.
__device__ void finish_step(const DevPool& p, const StepFinish& f, const long long* __restrict__ R) {
  int32_t sid = f.sid_dev ? (int32_t)*f.sid_dev : f.sid;
  const int status = (int)R[R_STATUS];
  if (f.turn_end && sid >= 0 && sid < p.S && status != LV_RESIDENT_FAILED) {
    lv_session_state st = p.sess[sid];
    lv_event x{};
    x.kind = LV_EV_TURN_END;
    x.sid = sid;
    x.t_us = f.now_us;
    x.a = f.audio_us;
    x.b = f.units;
    apply_event(p, st, x);
    p.sess[sid] = st;
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_EVENTS]), 1ull);
  }
  if (f.preload && status == LV_RESIDENT_DONE) {
    p.sess[sid].protect_until_us = f.now_us + p.protect_us;   // warmed KV (Section 5.2)
    atomicAdd(reinterpret_cast<unsigned long long*>(&p.ctl[C_PRELOADS]), 1ull);
  }
  if (f.out) {
    lv_resident_result r;
    r.k = R[R_K];
    r.n_found = R[R_FOUND];
    r.n_victims = R[R_N_OUT];
    r.n_loaded = R[R_N_IN];
    r.n_appended = (int32_t)R[R_APPENDED];
    r.status = status;
    r.sid = sid;
    *f.out = r;
  }
}

// ----------------------------------------------------------------- evict
// lv_evict: up to k victims by the normal order (no fallback tier), fewer when
// there are fewer candidates (GATE_EVICT); nothing is loaded.
__global__ void k_evict_prepare(long long k, long long* __restrict__ R) {
  pdl_entry();
  if (threadIdx.x != 0) return;
  R[R_K_SELECT] = k;
  R[R_N_OUT] = 0;
  R[R_N_IN] = 0;
  R[R_STATUS] = LV_RESIDENT_DONE;
  R[R_K] = k;
  R[R_GATE] = 1;
  R[R_APPENDED] = 0;
  R[R_FOUND] = 0;
  R[R_SID] = -1;
}


// ------------------------------------------------------------------ turn
// lv_turn's pick: CTA c reports whether candidate c has a block in the host tier.
__global__ void __launch_bounds__(kCensusThreads)
k_pick_scan(DevPool p, const int32_t* __restrict__ cand, int32_t* __restrict__ hit) {
  pdl_entry();
  const int32_t s = cand[blockIdx.x];
  int any = 0;
  if (s >= 0 && s < p.S) {
    const int32_t nb = nblocks_of(p, s);
    const int32_t* row = p.table + (size_t)s * p.maxB;
    for (int32_t b = threadIdx.x; b < nb && !any; b += kCensusThreads) any = row[b] <= -2;
  }
  any = __syncthreads_or(any);
  if (threadIdx.x == 0) hit[blockIdx.x] = any;
}

// ------------------------------------------------------------- checksums
constexpr int kSumThreads = 256;
constexpr int kSumUnroll = 4;
constexpr int kSumBatch = 4;      // sub-pages taken from the cursor at a time

// Unit u = (page i, sub-page j); the sub-page's words are q0 + k (q0 = j*P/8).
// Each thread keeps kSumUnroll 16-byte loads in flight; the per-unit partial sum
// goes to sums[i] with one atomic add (addition mod 2^64 is order-free).
__global__ void __launch_bounds__(kSumThreads)
k_checksum(DevPool p, const int32_t* __restrict__ pages, long long n, unsigned long long* __restrict__ sums,
           unsigned long long* __restrict__ cursor) {
  __shared__ unsigned long long warp_part[kSumThreads / 32];
  __shared__ long long s_next;
  const long long units = n * p.J;
  const int nvec = (int)(p.P >> 4);                   // 16-byte vectors per sub-page
  // units come from a shared cursor, kSumBatch at a time, the next batch fetched while
  // the current one is read: a CTA that starts late (its SM held by other work) takes
  // fewer units instead of holding up the end of the call
  // (thread 0 keeps the fetched index in a register and publishes it only at the end
  // of the batch, so that its warp does not wait for the atomic's result meanwhile)
  if (threadIdx.x == 0) s_next = (long long)atomicAdd(cursor, (unsigned long long)kSumBatch);
  __syncthreads();
  for (long long b = s_next; b < units; b = s_next) {
    unsigned long long fetched = 0;
    if (threadIdx.x == 0) fetched = atomicAdd(cursor, (unsigned long long)kSumBatch);
    const long long b_end = b + kSumBatch < units ? b + kSumBatch : units;
    for (long long u = b; u < b_end; ++u) {
      const long long i = u / p.J;
      const int j = (int)(u % p.J);
      const int32_t pg = pages[i];
      const bool ok = pg >= 0 && pg < p.hbm_pages;
      unsigned long long acc = 0;
      if (ok) {
        const ulonglong2* src = reinterpret_cast<const ulonglong2*>(p.kv[j] + (size_t)pg * p.P);
        const unsigned long long q0 = (unsigned long long)j * (unsigned long long)(p.P >> 3);
        for (int base = threadIdx.x; base < nvec; base += kSumThreads * kSumUnroll) {
          ulonglong2 r[kSumUnroll];
#pragma unroll
          for (int k = 0; k < kSumUnroll; ++k) {
            const int v = base + k * kSumThreads;
            if (v < nvec) r[k] = src[v];
          }
#pragma unroll
          for (int k = 0; k < kSumUnroll; ++k) {
            const int v = base + k * kSumThreads;
            if (v < nvec) {
              const unsigned long long q = q0 + 2ull * (unsigned long long)v;   // word index of r.x
              acc += r[k].x * (2ull * q + 1ull) + r[k].y * (2ull * q + 3ull);
            }
          }
        }
      } else if (j == 0 && threadIdx.x == 0) {
        set_error(p.ctl, LV_ERR_BOUNDS, i);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc += __shfl_down_sync(0xffffffffu, acc, o);
      if ((threadIdx.x & 31) == 0) warp_part[threadIdx.x >> 5] = acc;
      __syncthreads();
      if (threadIdx.x == 0) {
        unsigned long long t = 0;
#pragma unroll
        for (int w = 0; w < kSumThreads / 32; ++w) t += warp_part[w];
        if (ok) atomicAdd(&sums[i], t);
      }
      __syncthreads();
    }
    if (threadIdx.x == 0) s_next = (long long)fetched;   // every thread has read b
    __syncthreads();
  }
}

// ----------------------------------------------------------------- views
__global__ void __launch_bounds__(kCensusThreads)
k_counts(DevPool p, int32_t* __restrict__ hbm, int32_t* __restrict__ host) {
  const int32_t s = blockIdx.x;
  const int32_t nb = nblocks_of(p, s);
  const int32_t* row = p.table + (size_t)s * p.maxB;
  long long a = 0, h = 0;
  for (int32_t b = threadIdx.x; b < nb; b += kCensusThreads) {
    const int32_t e = row[b];
    a += e >= 0;
    h += e <= -2;
  }
  long long ta, th;
  block_excl_scan<kCensusThreads>(a, &ta);
  block_excl_scan<kCensusThreads>(h, &th);
  if (threadIdx.x == 0) {
    if (hbm) hbm[s] = (int32_t)ta;
    if (host) host[s] = (int32_t)th;
  }
}

__global__ void __launch_bounds__(kCensusThreads)
k_blocks(DevPool p, int32_t sid, int32_t where, int32_t* __restrict__ out, long long* count) {
  const int32_t nb = nblocks_of(p, sid);
  const int32_t* row = p.table + (size_t)sid * p.maxB;
  long long run = 0;
  for (int32_t q0 = 0; q0 < nb; q0 += kCensusThreads) {
    const int32_t b = q0 + threadIdx.x;
    long long flag = 0;
    if (b < nb) flag = where == 0 ? row[b] >= 0 : row[b] <= -2;
    long long chunk;
    const long long pos = run + block_excl_scan<kCensusThreads>(flag, &chunk);
    if (flag) out[pos] = b;
    run += chunk;
  }
  if (threadIdx.x == 0 && count) *count = run;
}

inline unsigned blocks_for(long long n, int threads, long long cap) {
  long long b = (n + threads - 1) / threads;
  if (b < 1) b = 1;
  if (b > cap) b = cap;
  return (unsigned)b;
}

}  // namespace

// ======================================================== launch wrappers
cudaError_t launch_import(const DevPool& p, const int32_t* placement, const int32_t* ctx,
                          cudaStream_t s) {
  k_import<<<blocks_for((long long)p.S * p.maxB, 256, 4096), 256, 0, s>>>(p, placement, ctx);
  return cudaGetLastError();
}

cudaError_t launch_check_budget(const DevPool& p, cudaStream_t s) {
  k_check_budget<<<1, 1, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_session_set(const DevPool& p, const lv_session_state* in, int32_t first,
                               int32_t n, cudaStream_t s) {
  k_session_set<<<blocks_for(n, 256, 1 << 20), 256, 0, s>>>(p, in, first, n);
  return cudaGetLastError();
}

thread_local std::vector<LaunchRecord>* t_recorder = nullptr;

void set_launch_recorder(std::vector<LaunchRecord>* rec) { t_recorder = rec; }

cudaError_t replay_launches(const std::vector<LaunchRecord>& recs, cudaStream_t s) {
  for (const LaunchRecord& r : recs) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = r.grid;
    cfg.blockDim = r.block;
    cfg.dynamicSmemBytes = r.smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = r.pdl ? 1 : 0;
    const cudaError_t e = cudaLaunchKernelExC(&cfg, r.func, const_cast<void**>(r.args.data()));
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

// A launch that lets the kernel be scheduled while the previous kernel on `s`
// still runs; the kernel must begin with pdl_entry().  With a recorder set on this
// thread the launch is recorded (its arguments converted to the kernel's parameter
// types and kept) instead of issued.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, unsigned block, size_t smem,
                       cudaStream_t s, Args&&... args) {
  if (t_recorder) {
    using Values = std::tuple<std::decay_t<KArgs>...>;
    auto values = std::make_shared<Values>(std::forward<Args>(args)...);
    LaunchRecord r{reinterpret_cast<const void*>(kernel), grid, dim3(block), smem, true, values, {}};
    std::apply([&r](auto&... x) { (r.args.push_back(static_cast<void*>(&x)), ...); }, *values);
    t_recorder->push_back(std::move(r));
    return cudaSuccess;
  }
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

cudaError_t launch_events(const DevPool& p, const lv_event* ev, int64_t n, cudaStream_t s) {
  k_events<<<blocks_for(p.S, kEventThreads, 1 << 20), kEventThreads, 0, s>>>(p, ev, n);
  return cudaGetLastError();
}

cudaError_t launch_select(const DevPool& p, int64_t now_us, int64_t k, bool fallback,
                          lv_victim* out, long long* count_dev, cudaStream_t s, int /*num_sms*/,
                          const long long* k_dev) {
  cudaError_t e = launch_pdl(k_rank_census, (unsigned)p.S, kCensusThreads, 0, s, p, (long long)now_us,
                             fallback, k_dev);
  if (e != cudaSuccess) return e;
  if (p.S > kEmitScanMax) {
    const dim3 grid((unsigned)((p.S + kPrefixTile - 1) / kPrefixTile),
                    (unsigned)((p.S + kPrefixChunk - 1) / kPrefixChunk));
    e = launch_pdl(k_rank_prefix, grid, kPrefixTile, 0, s, p, k_dev);
    if (e != cudaSuccess) return e;
  }
  e = launch_pdl(k_rank_emit, (unsigned)p.S, kEmitThreads, 0, s, p, (long long)k, k_dev, fallback,
                 count_dev, out);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}


cudaError_t launch_alloc(const DevPool& p, bool hbm, int64_t n, int32_t* out, cudaStream_t s,
                         bool injected_fail) {
  k_alloc<<<1, kAllocThreads, 0, s>>>(p, hbm, n, out, injected_fail);
  return cudaGetLastError();
}

cudaError_t launch_alloc_out(const DevPool& p, const lv_victim* v, int64_t n, int32_t* out,
                             cudaStream_t s, bool injected_fail) {
  if (n <= 0) return cudaSuccess;
  k_alloc_out<<<1, kAllocThreads, 0, s>>>(p, v, n, out, injected_fail);
  return cudaGetLastError();
}

cudaError_t launch_swap_out(const DevPool& p, const lv_victim* v, const int32_t* slots, int64_t n,
                            lv_remap_entry* commit, cudaStream_t s, int num_sms, const EventPair* ev) {
  const long long units = (long long)n * p.J;
  if (ev) cudaEventRecord(ev->start, s);
  k_swap_out<<<blocks_for(units, 1, (long long)num_sms * 8), kCopyThreads, 0, s>>>(
      p, v, slots, n, commit);
  if (ev) cudaEventRecord(ev->end, s);
  return cudaGetLastError();
}

cudaError_t launch_swap_in(const DevPool& p, int32_t sid, const int32_t* blks, const int32_t* pages,
                           int64_t n, lv_remap_entry* commit, cudaStream_t s, int num_sms,
                           const EventPair* ev) {
  const long long units = (long long)n * p.J;
  if (ev) cudaEventRecord(ev->start, s);
  k_swap_in<<<blocks_for(units, 1, (long long)num_sms * 8), kCopyThreads, 0, s>>>(
      p, sid, blks, pages, n, commit);
  if (ev) cudaEventRecord(ev->end, s);
  return cudaGetLastError();
}

cudaError_t launch_exchange(const DevPool& p, const lv_victim* v, int64_t n_out, int32_t sid,
                            const int32_t* blks, int64_t n_in, int32_t* slots, int32_t* pages,
                            int4* tasks, long long* n_tasks, int32_t epoch,
                            unsigned long long* page_tag, cudaStream_t s, int copy_ctas,
                            const long long* counts_dev, long long max_units, const EventPair* ev,
                            const long long* sid_dev, const CopyOffload* off, int gate,
                            long long* cursor, const StepFinish* fin) {
  long long* R = gate != GATE_NONE ? const_cast<long long*>(counts_dev) - R_N_OUT : nullptr;
  if (R) cursor = R + R_CURSOR;
  const StepFinish no_fin{};
  cudaError_t le = launch_pdl(k_exchange_plan, 1, kPlanThreads, 0, s, p, v, (long long)n_out, sid,
                              blks, (long long)n_in, slots, pages, tasks, n_tasks, epoch, page_tag,
                              counts_dev, sid_dev, R, gate, cursor, fin && R ? *fin : no_fin);
  if (le != cudaSuccess) return le;
  const long long units = counts_dev ? max_units : (n_out + n_in) * (long long)p.J;
  cudaStream_t cs = s;
  if (off) {
    cudaError_t e = cudaEventRecord(off->planned, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(off->stream, off->planned, 0);
    if (e != cudaSuccess) return e;
    cs = off->stream;
  }
  if (ev) cudaEventRecord(ev->start, cs);
  else if (off && off->started) cudaEventRecord(off->started, cs);
  const unsigned grid = blocks_for(units, 1, copy_ctas);
  if (p.xstages > 0) {
    const size_t smem = (size_t)p.xstages * 2 * p.P;
    if (off || ev) {
      k_exchange_copy_tma<<<grid, kStageThreads, smem, cs>>>(p, tasks, n_tasks, cursor);
    } else {
      le = launch_pdl(k_exchange_copy_tma, grid, kStageThreads, smem, cs, p, (const int4*)tasks,
                      (const long long*)n_tasks, cursor);
      if (le != cudaSuccess) return le;
    }
  } else if (off || ev) {   // after an event wait or record: an ordinary launch
    k_exchange_copy<<<grid, kCopyThreads, 0, cs>>>(p, tasks, n_tasks, cursor);
  } else {
    le = launch_pdl(k_exchange_copy, grid, kCopyThreads, 0, cs, p, (const int4*)tasks,
                    (const long long*)n_tasks, cursor);
    if (le != cudaSuccess) return le;
  }
  if (ev) cudaEventRecord(ev->end, cs);
  else if (off && off->finished) cudaEventRecord(off->finished, cs);
  if (off) {
    const cudaError_t e = cudaEventRecord(off->copied, cs);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

cudaError_t launch_make_resident(const DevPool& p, const ResidentScratch& rs, int32_t sid,
                                 int64_t now_us, int32_t append_tokens, bool preload,
                                 int64_t max_load, int32_t epoch, cudaStream_t s, int copy_ctas,
                                 lv_resident_result* result, const EventPair* ev,
                                 const long long* sid_dev, const CopyOffload* off,
                                 const unsigned long long* load_keys, bool turn_end,
                                 int64_t audio_us, int64_t units, const TurnStart* ts) {
  long long* R = rs.words;
  const TurnStart none{};
  cudaError_t e = launch_pdl(k_resident_prepare, 1, kCensusThreads, 0, s, p, sid, append_tokens,
                             preload, (long long)max_load, rs.blocks, R, sid_dev, ts ? *ts : none);
  if (e != cudaSuccess) return e;
  if (load_keys) {
    e = launch_pdl(k_order_loads, blocks_for(p.maxB, kOrderThreads / 32, 1ll << 30), kOrderThreads, 0,
                   s, (const long long*)R, (const int32_t*)rs.blocks, load_keys, rs.loads);
    if (e != cudaSuccess) return e;
  }
  e = launch_select(p, now_us, 0, !preload, rs.victims, nullptr, s, 0, R + R_K_SELECT);
  if (e != cudaSuccess) return e;
  const long long max_units = ((long long)p.budget + p.maxB) * p.J;
  // the step's end (turn end, preload protection, result): in the plan kernel when no
  // append follows it, else in a kernel of its own after the append
  const StepFinish fin{true, sid, sid_dev, (long long)now_us, preload, turn_end, (long long)audio_us,
                       (long long)units, result};
  e = launch_exchange(p, rs.victims, 0, sid, load_keys ? rs.loads : rs.blocks, 0, rs.slots, rs.pages,
                      rs.tasks, R + R_N_TASKS, epoch, p.page_tag, s, copy_ctas, R + R_N_OUT, max_units,
                      ev, sid_dev, off, preload ? GATE_PRELOAD : GATE_RESIDENT, nullptr,
                      append_tokens > 0 ? nullptr : &fin);
  if (e != cudaSuccess) return e;
  if (append_tokens > 0) {   // the growth, then the step's end in the same kernel
    e = launch_append(p, sid, append_tokens, rs.append, reinterpret_cast<int32_t*>(R + R_APPENDED), s,
                      R + R_GATE, sid_dev, &fin, R);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

cudaError_t launch_evict(const DevPool& p, const ResidentScratch& rs, int64_t now_us, int64_t k,
                         int32_t epoch, cudaStream_t s, int copy_ctas, lv_resident_result* result,
                         const EventPair* ev, const CopyOffload* off) {
  long long* R = rs.words;
  cudaError_t e = launch_pdl(k_evict_prepare, 1, 32, 0, s, (long long)k, R);
  if (e != cudaSuccess) return e;
  e = launch_select(p, now_us, 0, false, rs.victims, nullptr, s, 0, R + R_K_SELECT);
  if (e != cudaSuccess) return e;
  const long long max_units = (long long)p.budget * p.J;
  const StepFinish fin{true, -1, nullptr, (long long)now_us, false, false, 0, 0, result};
  e = launch_exchange(p, rs.victims, 0, -1, rs.blocks, 0, rs.slots, rs.pages, rs.tasks,
                      R + R_N_TASKS, epoch, p.page_tag, s, copy_ctas, R + R_N_OUT, max_units, ev,
                      nullptr, off, GATE_EVICT, nullptr, &fin);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_turn(const DevPool& p, const ResidentScratch& rs, int32_t sid, const int32_t* cand,
                        int32_t n_cand, int64_t now_us, int32_t append_tokens, int64_t audio_us,
                        int64_t units, int32_t epoch, cudaStream_t s, int copy_ctas,
                        lv_resident_result* result, const EventPair* ev, const CopyOffload* off,
                        const unsigned long long* load_keys) {
  long long* R = rs.words;
  cudaError_t e0 = cudaSuccess;
  if (sid < 0) {
    e0 = launch_pdl(k_pick_scan, (unsigned)n_cand, kCensusThreads, 0, s, p, cand, rs.hits);
    if (e0 != cudaSuccess) return e0;
  }
  // turn start (in the prepare kernel), make resident, then (in its finish kernel)
  // LV_EV_TURN_END
  const TurnStart ts{true, cand, n_cand, rs.hits, (long long)now_us};
  cudaError_t e = launch_make_resident(p, rs, sid, now_us, append_tokens, false, -1, epoch, s,
                                       copy_ctas, result, ev, R + R_SID, off, load_keys, true,
                                       audio_us, units, &ts);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// Zeroes `words` 32-bit words at p, which may be device memory or the device alias of
// mapped page-locked host memory (a kernel, so that either works).
__global__ void k_zero(uint32_t* __restrict__ q, long long words) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < words;
       i += (long long)gridDim.x * blockDim.x)
    q[i] = 0u;
}

cudaError_t launch_zero(void* q, int64_t bytes, cudaStream_t s) {
  const long long words = (long long)(bytes / 4);
  if (words <= 0) return cudaSuccess;
  k_zero<<<blocks_for(words, 256, 1024), 256, 0, s>>>(static_cast<uint32_t*>(q), words);
  return cudaGetLastError();
}

cudaError_t launch_checksums(const DevPool& p, const int32_t* pages, int64_t n,
                             unsigned long long* sums, unsigned long long* cursor, cudaStream_t s,
                             int ctas) {
  if (n <= 0) return cudaSuccess;
  k_checksum<<<blocks_for(n * p.J, kSumBatch, ctas), kSumThreads, 0, s>>>(p, pages, n, sums, cursor);
  return cudaGetLastError();
}

cudaError_t launch_selftest_wait(const DevPool& p, long long limit_ns, cudaStream_t s) {
  k_selftest_wait<<<1, 32, 0, s>>>(p.ctl, limit_ns);
  return cudaGetLastError();
}

cudaError_t launch_tasks_out(const DevPool& p, const lv_victim* v, const int32_t* slots, int64_t n,
                             int4* tasks, lv_remap_entry* commit, cudaStream_t s) {
  k_tasks_out<<<blocks_for(n, 256, 1ll << 30), 256, 0, s>>>(p, v, slots, n, tasks, commit);
  return cudaGetLastError();
}

cudaError_t launch_tasks_in(const DevPool& p, int32_t sid, const int32_t* blks, const int32_t* pages,
                            int64_t n, int4* tasks, lv_remap_entry* commit, cudaStream_t s) {
  k_tasks_in<<<blocks_for(n, 256, 1ll << 30), 256, 0, s>>>(p, sid, blks, pages, n, tasks, commit);
  return cudaGetLastError();
}

// About 48 KiB of stages per CTA, two CTAs per SM: on GB300 three 16 KiB stages per CTA
// moved 4096 scattered thinker pages at 6.82-6.94 TB/s (read + write), against 6.2-6.4
// with eight stages and one CTA per SM, and 5.5 with two stages.
int stage_count(const DevPool& p) {
  int st = p.stages > 0 ? p.stages : (int)((48 * 1024) / p.P);
  if (st < 3) st = 3;
  if (st > kMaxStages) st = kMaxStages;
  if ((long long)st * p.P > 227 * 1024) st = (int)((227 * 1024) / p.P);
  return st < 2 ? 2 : st;
}

cudaError_t configure_stage_kernels(const DevPool& p) {
  const int smem = stage_count(p) * (int)p.P;
  cudaError_t e = cudaFuncSetAttribute(k_stage_tasks<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_stage_tasks<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
}

int exchange_stage_limit(long long P) {
  const long long per = 2 * P;
  long long n = (227ll * 1024) / per;
  if (n > kXStageMax) n = kXStageMax;
  return n >= 2 ? (int)n : 0;
}

cudaError_t configure_exchange_tma(const DevPool& p) {
  if (p.xstages <= 0) return cudaSuccess;
  return cudaFuncSetAttribute(k_exchange_copy_tma, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)((size_t)p.xstages * 2 * p.P));
}

cudaError_t launch_stage(const DevPool& p, bool pack, const int4* tasks, int64_t t_begin, int64_t t_end,
                         uint8_t* staging, cudaStream_t s, int ctas, const EventPair* ev, bool tma) {
  if (t_end <= t_begin) return cudaSuccess;
  const long long units = (t_end - t_begin) * (long long)p.J;
  if (ev) cudaEventRecord(ev->start, s);
  if (tma) {
    const int stages = stage_count(p);
    const size_t smem = (size_t)stages * p.P;
    const unsigned grid = blocks_for(units, 1, ctas);
    if (pack)
      k_stage_tasks<true><<<grid, kStageThreads, smem, s>>>(p, tasks, t_begin, t_end, staging, stages);
    else
      k_stage_tasks<false><<<grid, kStageThreads, smem, s>>>(p, tasks, t_begin, t_end, staging, stages);
  } else {
    const unsigned grid = blocks_for(units, 1, 4ll * ctas);
    if (pack)
      k_stage_tasks_lsu<true><<<grid, kCopyThreads, 0, s>>>(p, tasks, t_begin, t_end, staging);
    else
      k_stage_tasks_lsu<false><<<grid, kCopyThreads, 0, s>>>(p, tasks, t_begin, t_end, staging);
  }
  if (ev) cudaEventRecord(ev->end, s);
  return cudaGetLastError();
}

cudaError_t launch_tasks_pages(const DevPool& p, const int32_t* pages, int64_t n, bool pack, int4* tasks,
                               cudaStream_t s) {
  k_tasks_pages<<<blocks_for(n, 256, 1ll << 30), 256, 0, s>>>(p, pages, n, pack, tasks);
  return cudaGetLastError();
}

cudaError_t launch_exchange_plan(const DevPool& p, const lv_victim* v, int64_t n_out, int32_t sid,
                                 const int32_t* blks, int64_t n_in, int32_t* slots, int32_t* pages,
                                 int4* tasks, long long* n_tasks, int32_t epoch,
                                 unsigned long long* page_tag, cudaStream_t s) {
  k_exchange_plan<<<1, kPlanThreads, 0, s>>>(p, v, n_out, sid, blks, n_in, slots, pages, tasks,
                                             n_tasks, epoch, page_tag, nullptr, nullptr, nullptr,
                                             (int)GATE_NONE, nullptr, StepFinish{});
  return cudaGetLastError();
}

cudaError_t launch_remap(const DevPool& p, const lv_remap_entry* e, int64_t n, int32_t epoch,
                         cudaStream_t s, int num_sms, int per_thread) {
  if (n <= 0) return cudaSuccess;
  // one entry per thread while the GPU holds every thread at once; beyond that, up
  // to four entries per thread so that their reads overlap
  const long long resident = (long long)(num_sms > 0 ? num_sms : 1) * 2048;
  int E = per_thread;
  if (E != 1 && E != 2 && E != 4) E = n <= resident ? 1 : (n <= 2 * resident ? 2 : 4);
  const unsigned grid = blocks_for((n + E - 1) / E, kRemapThreads, 1ll << 30);
  if (E == 1) k_remap<1><<<grid, kRemapThreads, 0, s>>>(p, e, n, epoch);
  else if (E == 2) k_remap<2><<<grid, kRemapThreads, 0, s>>>(p, e, n, epoch);
  else k_remap<4><<<grid, kRemapThreads, 0, s>>>(p, e, n, epoch);
  cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  // the release pass over both tiers' owner words (8 quads of 4 per bitmap word)
  const long long qh = (long long)((p.hbm_pages + 31) / 32) * 8;
  const long long qo = (long long)((p.host_pages + 31) / 32) * 8;
  const long long cap = (long long)(num_sms > 0 ? num_sms : 1) * 8;
  const long long per_cta = (long long)kReleaseThreads * kReleaseUnroll;
  long long rg = (qh + qo + per_cta - 1) / per_cta;
  if (rg > cap) rg = cap;
  err = launch_pdl(k_release, dim3((unsigned)rg), kReleaseThreads, 0, s, p, qh, qo);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

cudaError_t launch_cancel(const DevPool& p, const int32_t* locs, int64_t n, cudaStream_t s) {
  k_cancel<<<blocks_for(n, 256, 1ll << 30), 256, 0, s>>>(p, locs, n);
  return cudaGetLastError();
}

cudaError_t launch_append(const DevPool& p, int32_t sid, int32_t n_tokens, int32_t* pages,
                          int32_t* count, cudaStream_t s, const long long* gate,
                          const long long* sid_dev, const StepFinish* fin, const long long* R) {
  const StepFinish none{};
  const cudaError_t e = launch_pdl(k_append, 1, kAllocThreads, 0, s, p, sid, n_tokens, pages, count,
                                   gate, sid_dev, fin ? *fin : none, R);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_counts(const DevPool& p, int32_t* hbm, int32_t* host, cudaStream_t s) {
  k_counts<<<p.S, kCensusThreads, 0, s>>>(p, hbm, host);
  return cudaGetLastError();
}

cudaError_t launch_blocks(const DevPool& p, int32_t sid, int32_t where, int32_t* out,
                          long long* count, cudaStream_t s) {
  k_blocks<<<1, kCensusThreads, 0, s>>>(p, sid, where, out, count);
  return cudaGetLastError();
}

}  // namespace lv
