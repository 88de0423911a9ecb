// The preload controller of Section 5.2 (see include/lv.h for its readings): host
// code that decides when a speech-triggered preload may run and drives the pool's
// own calls -- ranking, exchange (the evictions), swap-in (reserve and fill),
// remap (the deferred commit), cancel, and the monitor's PRELOADED / UNPROTECT
// events.  It keeps a modelled host->device link, each session's speech-to-turn
// lead, the waiting and pending preloads, and a log of its decisions.
#include <algorithm>
#include <cstring>
#include <map>
#include <new>
#include <set>
#include <utility>
#include <vector>

#include "lv_internal.cuh"

struct lv_controller {
  lv_pool* pool = nullptr;
  int64_t bw = 1, lead_prior = 0, cap = -1;
  int32_t mode = LV_MODE_AUTO;
  int32_t S = 0, maxB = 0;
  int64_t page_bytes = 0, budget = 0, host_pages = 0;
  int64_t link_free_at = 0;
  std::map<int32_t, std::pair<int64_t, int64_t>> lead;   // sid -> (EMA, samples)
  std::map<int32_t, int64_t> speech_t;                    // sid -> speech start before its turn
  struct Wait {
    int64_t t_pred;
    int64_t refused;
  };
  std::map<int32_t, Wait> waiting;
  struct Pending {
    int64_t finish;
    int64_t n;
    int32_t* pages;            // device [n]: the reserved HBM pages
    lv_remap_entry* commit;    // device [n]: their commit entries
  };
  std::map<int32_t, Pending> pending;
  std::set<int32_t> completed;
  lv_controller_counters ctr{};
  std::vector<lv_controller_record> log;
  std::vector<int32_t> log_data;
};

namespace {

#define CTL_TRY(expr)                 \
  do {                                \
    const lv_status _s = (expr);      \
    if (_s != LV_OK) return _s;       \
  } while (0)

int64_t duration_us(const lv_controller* c, int64_t pages) {
  const int64_t b = pages * c->page_bytes;
  return (b + c->bw - 1) / c->bw;
}

int64_t lead_of(const lv_controller* c, int32_t sid) {
  auto it = c->lead.find(sid);
  return (it != c->lead.end() && it->second.second > 0) ? it->second.first : c->lead_prior;
}

void record(lv_controller* c, int32_t kind, int32_t sid, int64_t start = 0, int64_t finish = 0,
            int64_t deadline = 0, int64_t n = 0, const int32_t* data = nullptr, int64_t n_data = 0) {
  lv_controller_record r{};
  r.kind = kind;
  r.sid = sid;
  r.start_us = start;
  r.finish_us = finish;
  r.deadline_us = deadline;
  r.n = n;
  r.data_offset = (int64_t)c->log_data.size();
  c->log.push_back(r);
  if (n_data > 0) c->log_data.insert(c->log_data.end(), data, data + n_data);
}

// The session's blocks in the host tier, ascending (a host wait).
lv_status host_blocks(lv_controller* c, int32_t sid, lv_stream s, std::vector<int32_t>* out) {
  out->assign((size_t)c->maxB, 0);
  int64_t n = 0;
  CTL_TRY(lv_session_blocks(c->pool, sid, 1, out->data(), &n, s));
  CTL_TRY(lv_sync(c->pool, s));
  out->resize((size_t)n);
  return LV_OK;
}

void release(lv_controller::Pending& p, cudaStream_t s) {
  if (p.pages) cudaFreeAsync(p.pages, s);
  if (p.commit) cudaFreeAsync(p.commit, s);
  p.pages = nullptr;
  p.commit = nullptr;
}

lv_status try_admit(lv_controller* c, int32_t sid, int64_t t, lv_stream s) {
  auto wit = c->waiting.find(sid);
  std::vector<int32_t> blks;
  CTL_TRY(host_blocks(c, sid, s, &blks));
  const int64_t n = (int64_t)blks.size();
  if (n == 0) {
    c->waiting.erase(wit);
    return LV_OK;
  }
  const int64_t start = std::max(t, c->link_free_at);
  const int64_t finish = start + duration_us(c, n);
  if (finish > wit->second.t_pred) {
    ++wit->second.refused;
    return LV_OK;
  }
  lv_stats st;
  CTL_TRY(lv_get_stats(c->pool, &st, s));
  const int64_t k = std::max<int64_t>(0, n - (st.hbm_budget_pages - st.hbm_allocated));
  const int64_t host_free = st.host_pages - st.host_allocated;
  if (k > host_free - c->maxB) {
    ++wit->second.refused;
    return LV_OK;
  }
  if (k > 0) {
    std::vector<lv_victim> v((size_t)k);
    int64_t nv = 0;
    CTL_TRY(lv_select_victims(c->pool, t, k, 0, v.data(), k, &nv, s));
    CTL_TRY(lv_sync(c->pool, s));
    if (nv < k) {
      ++wit->second.refused;
      return LV_OK;
    }
    record(c, LV_CTL_EVICTED, sid, 0, 0, 0, k, reinterpret_cast<const int32_t*>(v.data()), 3 * k);
    CTL_TRY(lv_swap_exchange(c->pool, v.data(), k, 0, nullptr, 0, nullptr, nullptr, c->mode, s));
    c->ctr.victims += k;
  }
  cudaStream_t cs = static_cast<cudaStream_t>(s);
  lv_controller::Pending p{finish, n, nullptr, nullptr};
  if (cudaMallocAsync((void**)&p.pages, (size_t)n * sizeof(int32_t), cs) != cudaSuccess ||
      cudaMallocAsync((void**)&p.commit, (size_t)n * sizeof(lv_remap_entry), cs) != cudaSuccess) {
    cudaGetLastError();
    release(p, cs);
    return LV_ERR_OOM;
  }
  lv_status r = lv_swap_in(c->pool, sid, blks.data(), n, p.pages, p.commit, c->mode, s);
  std::vector<int32_t> pages_h((size_t)n);
  if (r == LV_OK) r = lv_sync(c->pool, s);
  if (r == LV_OK && cudaMemcpy(pages_h.data(), p.pages, (size_t)n * sizeof(int32_t),
                               cudaMemcpyDeviceToHost) != cudaSuccess)
    r = LV_ERR_CUDA;
  if (r != LV_OK) {
    release(p, cs);
    return r;
  }
  c->ctr.pages_in += n;
  c->link_free_at = finish;
  ++c->ctr.admitted;
  if (wit->second.refused) ++c->ctr.waited;
  const int64_t t_pred = wit->second.t_pred;
  c->waiting.erase(wit);
  c->pending[sid] = p;
  record(c, LV_CTL_ADMITTED, sid, start, finish, t_pred, n, pages_h.data(), n);
  return LV_OK;
}

// The protected sessions' resident pages above the cap: drop the oldest protections.
lv_status enforce_cap(lv_controller* c, int64_t now, lv_stream s) {
  if (c->cap < 0) return LV_OK;
  std::vector<lv_session_state> st((size_t)c->S);
  CTL_TRY(lv_session_get(c->pool, st.data(), 0, c->S, s));
  CTL_TRY(lv_sync(c->pool, s));
  std::vector<std::pair<int64_t, int32_t>> prot;
  for (int32_t q = 0; q < c->S; ++q)
    if (st[(size_t)q].protect_until_us > now) prot.emplace_back(st[(size_t)q].protect_until_us, q);
  if (prot.empty()) return LV_OK;
  std::sort(prot.begin(), prot.end());
  std::vector<int32_t> hbm((size_t)c->S);
  CTL_TRY(lv_session_counts(c->pool, hbm.data(), nullptr, s));
  CTL_TRY(lv_sync(c->pool, s));
  int64_t total = 0;
  for (const auto& x : prot) total += hbm[(size_t)x.second];
  std::vector<lv_event> drop;
  for (const auto& x : prot) {
    if (total <= c->cap) break;
    lv_event e{};
    e.kind = LV_EV_UNPROTECT;
    e.sid = x.second;
    e.t_us = now;
    drop.push_back(e);
    total -= hbm[(size_t)x.second];
  }
  if (drop.empty()) return LV_OK;
  CTL_TRY(lv_session_events(c->pool, drop.data(), (int64_t)drop.size(), s));
  for (const auto& e : drop) record(c, LV_CTL_UNPROTECTED, e.sid);
  return LV_OK;
}

lv_status complete(lv_controller* c, int32_t sid, lv_stream s) {
  auto it = c->pending.find(sid);
  lv_controller::Pending p = it->second;
  c->pending.erase(it);
  lv_status r = lv_remap(c->pool, p.commit, p.n, s);
  release(p, static_cast<cudaStream_t>(s));
  CTL_TRY(r);
  lv_event e{};
  e.kind = LV_EV_PRELOADED;
  e.sid = sid;
  e.t_us = p.finish;
  CTL_TRY(lv_session_events(c->pool, &e, 1, s));
  ++c->ctr.completed;
  c->completed.insert(sid);
  CTL_TRY(enforce_cap(c, p.finish, s));
  record(c, LV_CTL_COMPLETED, sid);
  return LV_OK;
}

}  // namespace

extern "C" {

lv_status lv_controller_create(lv_pool* pool, const lv_controller_desc* d, lv_controller** out) {
  if (!out) return LV_ERR_INVALID;
  *out = nullptr;
  if (!pool || !d || d->link_bytes_per_us < 1 || d->lead_prior_us < 0 || d->cap_pages < -1 ||
      d->reserved != 0)
    return LV_ERR_INVALID;
  const int32_t mode = d->mode & ~LV_MODE_ASYNC;
  if (mode != LV_MODE_AUTO && mode != LV_MODE_ZERO_COPY && mode != LV_MODE_STAGED) return LV_ERR_INVALID;
  lv_controller* c = new (std::nothrow) lv_controller();
  if (!c) return LV_ERR_OOM;
  c->pool = pool;
  c->bw = d->link_bytes_per_us;
  c->lead_prior = d->lead_prior_us;
  c->cap = d->cap_pages;
  c->mode = d->mode;
  lv::pool_shape(pool, &c->S, &c->maxB, &c->page_bytes, &c->budget, &c->host_pages);
  *out = c;
  return LV_OK;
}

lv_status lv_controller_destroy(lv_controller* c, lv_stream s) {
  if (!c) return LV_ERR_INVALID;
  lv_status r = LV_OK;
  for (auto& kv : c->pending) {
    if (r == LV_OK) r = lv_cancel(c->pool, kv.second.pages, kv.second.n, s);
    release(kv.second, static_cast<cudaStream_t>(s));
  }
  delete c;
  return r;
}

// Completes the preloads whose modelled transfer has finished (in finish order) and
// re-checks the waiting ones (in session order).
lv_status lv_controller_tick(lv_controller* c, int64_t t, lv_stream s) {
  if (!c) return LV_ERR_INVALID;
  try {
    std::vector<std::pair<int64_t, int32_t>> due;
    for (const auto& kv : c->pending)
      if (kv.second.finish <= t) due.emplace_back(kv.second.finish, kv.first);
    std::sort(due.begin(), due.end());
    for (const auto& x : due) CTL_TRY(complete(c, x.second, s));
    std::vector<int32_t> ids;
    for (const auto& kv : c->waiting) ids.push_back(kv.first);
    for (int32_t sid : ids) {
      auto it = c->waiting.find(sid);
      if (it == c->waiting.end()) continue;
      if (t >= it->second.t_pred) {
        c->waiting.erase(it);
        ++c->ctr.given_up;
        record(c, LV_CTL_GIVEN_UP, sid);
      } else {
        CTL_TRY(try_admit(c, sid, t, s));
      }
    }
    return LV_OK;
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_controller_speech(lv_controller* c, int32_t sid, int64_t t, lv_stream s) {
  if (!c || sid < 0 || sid >= c->S) return LV_ERR_INVALID;
  try {
    c->speech_t.emplace(sid, t);   // the first speech start before the turn counts
    if (c->pending.count(sid) || c->waiting.count(sid)) return LV_OK;
    std::vector<int32_t> blks;
    CTL_TRY(host_blocks(c, sid, s, &blks));
    if (blks.empty()) return LV_OK;
    c->waiting[sid] = lv_controller::Wait{c->speech_t[sid] + lead_of(c, sid), 0};
    return try_admit(c, sid, t, s);
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_controller_turn_begin(lv_controller* c, int32_t sid, int64_t t, lv_stream s) {
  if (!c || sid < 0 || sid >= c->S) return LV_ERR_INVALID;
  try {
    auto st = c->speech_t.find(sid);
    if (st != c->speech_t.end()) {   // one sample of the speech-to-turn lead
      const int64_t x = std::max<int64_t>(0, t - st->second);
      c->speech_t.erase(st);
      auto& l = c->lead[sid];
      l.first = l.second == 0 ? x : (3 * l.first + x) / 4;
      ++l.second;
    }
    auto w = c->waiting.find(sid);
    if (w != c->waiting.end()) {
      c->waiting.erase(w);
      ++c->ctr.given_up;
      record(c, LV_CTL_GIVEN_UP, sid);
    }
    auto p = c->pending.find(sid);
    if (p != c->pending.end()) {     // still in flight: the turn loads by itself
      const lv_status r = lv_cancel(c->pool, p->second.pages, p->second.n, s);
      release(p->second, static_cast<cudaStream_t>(s));
      c->pending.erase(p);
      CTL_TRY(r);
      ++c->ctr.cancelled;
      record(c, LV_CTL_CANCELLED, sid);
    }
    if (c->completed.erase(sid)) {
      std::vector<int32_t> blks;
      CTL_TRY(host_blocks(c, sid, s, &blks));
      if (blks.empty()) ++c->ctr.hits;
    }
    return LV_OK;
  } catch (const std::bad_alloc&) {
    return LV_ERR_OOM;
  }
}

lv_status lv_controller_turn_loaded(lv_controller* c, int64_t t, int64_t pages) {
  if (!c || pages < 0) return LV_ERR_INVALID;
  if (pages > 0) c->link_free_at = std::max(t, c->link_free_at) + duration_us(c, pages);
  return LV_OK;
}

lv_status lv_controller_records(lv_controller* c, lv_controller_record* records, int64_t capacity,
                                int64_t* n_records, int32_t* data, int64_t data_capacity,
                                int64_t* n_data) {
  if (!c || !n_records || !n_data) return LV_ERR_INVALID;
  *n_records = (int64_t)c->log.size();
  *n_data = (int64_t)c->log_data.size();
  if (capacity < *n_records || data_capacity < *n_data || (*n_records && !records) ||
      (*n_data && !data))
    return LV_ERR_INVALID;
  if (*n_records) std::memcpy(records, c->log.data(), c->log.size() * sizeof(lv_controller_record));
  if (*n_data) std::memcpy(data, c->log_data.data(), c->log_data.size() * sizeof(int32_t));
  c->log.clear();
  c->log_data.clear();
  return LV_OK;
}

lv_status lv_controller_counters_get(lv_controller* c, lv_controller_counters* out) {
  if (!c || !out) return LV_ERR_INVALID;
  *out = c->ctr;
  return LV_OK;
}

}  // extern "C"
