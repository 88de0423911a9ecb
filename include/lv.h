/*
 * lv.h -- C ABI of the interaction-aware KV swap path (liblv.so).
 *
 * A pool holds one engine stage's paged KV cache in two tiers: HBM (the
 * caller's per-layer K and V page arrays) and a page-locked host pool.  The
 * calls below rank resident blocks by predicted next use (Section 5.1, Eq. 4),
 * move blocks between the tiers (Section 5, Fig. 6: eviction to DRAM and
 * loading back, Section 5.2: speech-triggered preload) and commit the moves in
 * the block tables (Section 6, "Hierarchical KV cache manager": side tables on
 * sessions and blocks).
 *
 * Terms.  T tokens form a page (the paper's KV block); a page of one layer's K
 * or V is a sub-page of P = T*H*D*elem bytes laid out [T][H][D].  A page is
 * the allocation and eviction unit: all 2L sub-pages of T tokens share one
 * page id.  HBM sub-page j = 2*layer + kv (kv 0 = K, 1 = V) of page p lives at
 * hbm_kv[j] + p*P.  Host slot h holds a page as one contiguous run
 * [2L][P] at host_kv + h*2L*P.
 *
 * Block-table entries: e >= 0 is an HBM page id, e == -1 means "no block",
 * e <= -2 is host slot -(e + 2).
 *
 * Execution model.  Every call is asynchronous and ordered on the stream it
 * is given; argument checks that need no device data run at once and are the
 * return value.  Conditions found on the device (a bounds violation, a double
 * mapping, an exhausted tier) are recorded in a sticky per-pool error word that
 * lv_sync / lv_get_stats report; the kernels skip the offending item instead of
 * faulting, and no call traps, aborts or falls back to the CPU.  Nothing in the
 * library waits on the device except lv_sync, lv_get_stats and the readers
 * named as synchronous below.  Every call returns LV_ERR_INVALID for a NULL
 * pool or a NULL required pointer, LV_ERR_OOM when staging a host argument
 * needs memory that cannot be had, and LV_ERR_CUDA when a CUDA runtime call
 * fails; the comments below name the other statuses.
 *
 * Pointers.  Array arguments may point to device memory or to host memory.
 * Mapped page-locked host memory (any page-locked allocation under unified
 * addressing) is read and written by the kernels in place, over the host link;
 * the caller keeps such an input unchanged until the stream reaches the call.
 * A pageable host input is copied to the device before the call returns, and a
 * pageable host output is written by a copy queued on the stream.  Read any host
 * output after the stream has completed.
 * Calls that allocate from the same tier (swap-out: host slots; swap-in and
 * append: HBM pages) must be ordered with respect to each other.
 *
 * Threads.  A pool keeps host-side state (scratch alternation, pending
 * asynchronous copies, staging runs, timing records): calls on one pool must
 * not run concurrently from several host threads.  Distinct pools are
 * independent, and so is one pool per GPU.
 */
#ifndef LV_H
#define LV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef void* lv_stream;            /* a cudaStream_t; NULL = the legacy default stream */
typedef struct lv_pool lv_pool;     /* opaque */

typedef enum lv_status {
  LV_OK = 0,
  LV_ERR_INVALID = 1,     /* bad argument (size, alignment, pointer kind, range) */
  LV_ERR_OOM = 2,         /* a device or host allocation failed */
  LV_ERR_CUDA = 3,        /* a CUDA runtime call failed */
  LV_ERR_NO_HBM = 4,      /* HBM budget exhausted (device-detected) */
  LV_ERR_NO_HOST = 5,     /* host pool exhausted (device-detected) */
  LV_ERR_BOUNDS = 6,      /* an index outside the pool (device-detected) */
  LV_ERR_DOUBLE_MAP = 7,  /* a location or block committed twice (device-detected) */
  LV_ERR_BUDGET = 8,      /* more HBM pages allocated than the budget (device-detected) */
  LV_ERR_TIMEOUT = 9,     /* a bounded device wait ran out */
  LV_ERR_STATE = 10       /* a block is not where the call says it is (device-detected) */
} lv_status;

#define LV_ALL INT64_MAX             /* lv_select_victims: the whole victim order */

enum { LV_SUFFIX_FIRST = 0, LV_ASCENDING = 1 };        /* lv_pool_desc.within_order */
enum { LV_PLAY_PLAYBACK = 0, LV_PLAY_COUNTERS = 1 };   /* lv_pool_desc.t_play_mode */
enum { LV_MODE_AUTO = 0, LV_MODE_ZERO_COPY = 1, LV_MODE_STAGED = 2 };   /* swap modes */
/* lv_swap_exchange with LV_MODE_STAGED | LV_MODE_ASYNC: the call returns once its
   transfers are queued; its copy-engine transfers and unpacks overlap the
   caller's next calls.  A later asynchronous call waits for an earlier one's
   transfers of a direction only when it touches an HBM page or host slot that
   they may still be using.
   Until lv_join(pool, stream) the caller must not read or write the pool's KV
   arrays or host pool; calls that move or read KV bytes (other than another
   asynchronous staged exchange) and lv_sync join first by themselves. */
enum { LV_MODE_ASYNC = 16 };
enum { LV_SELECT_FALLBACK = 1 };                       /* lv_select_victims flags */
/* Victim order.  LV_POLICY_NEXT_USE: the paper's order (Section 5.1).
   LV_POLICY_LRU: the substrate's least-recently-used order that the paper
   compares against (Sections 2.3 and 5): candidates are all sessions that are
   not running, ranked by last use ascending (then session id ascending, suffix
   blocks first); speech, barge-in and preload protection are ignored. */
enum { LV_POLICY_NEXT_USE = 0, LV_POLICY_LRU = 1 };
/* Host-tier mode (lv_pool_desc.tiers).  The paper does not say whether a
   reloaded block keeps its host copy.  LV_TIERS_EXCLUSIVE: a block lives in
   one tier; its host slot is freed when it is committed back to HBM.
   LV_TIERS_INCLUSIVE: that slot stays allocated and owned by the block as its
   clean copy while the block's bytes are unchanged, so evicting the block
   again moves no bytes (lv_swap_out, lv_swap_exchange, lv_make_resident).  KV
   rows are written once, when their token is appended, so only the last,
   partially filled block of a session changes: lv_session_append and
   lv_make_resident drop that block's clean copy when they add rows to it.
   Clean copies are not reclaimed for other blocks: the host tier should hold
   a slot for every block (with fewer, an eviction fails with LV_ERR_NO_HOST as
   in the exclusive mode). */
enum { LV_TIERS_EXCLUSIVE = 0, LV_TIERS_INCLUSIVE = 1 };

/* session flag bits (lv_session_state.flags) */
enum {
  LV_RUNNING = 1,      /* the session's request executes: pinned running KV */
  LV_IMMEDIATE = 2,    /* speech start or barge-in seen: immediate reuse */
  LV_RESP_OPEN = 4,    /* the current reply is unfinished */
  LV_DONE_VALID = 8    /* t_done_us holds the completion time of the current reply */
};

/* monitor events (lv_event.kind) */
enum {
  LV_EV_TURN_BEGIN = 1,    /* the turn's request starts running */
  LV_EV_TURN_END = 2,      /* a = reply audio us, b = reply length in progress units */
  LV_EV_PLAYBACK = 3,      /* a = further us of the reply reported as played */
  LV_EV_SPEECH_START = 4,
  LV_EV_BARGE_IN = 5,      /* speech while the reply plays: unplayed audio discarded */
  LV_EV_SPEECH_STOP = 6,   /* the user input is complete */
  LV_EV_PRELOADED = 7,     /* a preload completed at t_us: protect the warmed KV */
  LV_EV_UNPROTECT = 8      /* the warmed KV's protection ends now (the cap, Section 5.2) */
};

typedef struct lv_pool_desc {
  int32_t num_layers;          /* L */
  int32_t num_kv_heads;        /* H */
  int32_t head_dim;            /* D */
  int32_t page_tokens;         /* T */
  int32_t elem_bytes;          /* bytes per K/V element (2 for bf16) */
  int32_t max_sessions;        /* S, 1..4096 */
  int32_t max_blocks;          /* block-table capacity per session, 1..65536 */
  int32_t within_order;        /* LV_SUFFIX_FIRST (default) or LV_ASCENDING */
  int64_t hbm_pages;           /* pages in each HBM sub-page array */
  int64_t hbm_budget_pages;    /* 0 < budget <= hbm_pages: allocated HBM pages at most */
  int64_t host_pages;          /* host pool slots */
  void* const* hbm_kv;         /* host array of 2L device pointers, each [hbm_pages][P],
                                  16-byte aligned; caller-owned, kept alive by the caller */
  void* host_kv;               /* page-locked host pool [host_pages][2L][P], or NULL: the
                                  library allocates (and frees) a mapped page-locked pool */
  int64_t reply_prior_us;      /* workload-level T_reply prior (>= 0) */
  int64_t protect_us;          /* preload protection window (>= 0) */
  int64_t unit_us;             /* progress-counter unit, 1..2^31 */
  int32_t t_play_mode;         /* LV_PLAY_PLAYBACK or LV_PLAY_COUNTERS */
  int32_t policy;              /* LV_POLICY_NEXT_USE (Section 5.1) or LV_POLICY_LRU */
  int32_t tiers;               /* LV_TIERS_EXCLUSIVE (default) or LV_TIERS_INCLUSIVE */
  int32_t reserved;            /* must be 0 */
} lv_pool_desc;

/* Per-session interaction state (72 bytes).  ctx_tokens is maintained by
   lv_pool_import and lv_session_append and ignored by lv_session_set. */
typedef struct lv_session_state {
  int32_t ctx_tokens;
  int32_t flags;               /* LV_RUNNING | LV_IMMEDIATE | LV_RESP_OPEN | LV_DONE_VALID */
  int64_t gen_us;              /* audio generated for the current reply */
  int64_t play_us;             /* audio of it reported as played */
  int64_t t_done_us;           /* completion time of the current reply (if LV_DONE_VALID) */
  int64_t reply_ema_us;        /* moving average of the reply interval */
  int32_t reply_n;             /* samples in it (0: the prior applies) */
  int32_t pad;
  int64_t reply_tokens;        /* current reply length in progress units */
  int64_t protect_until_us;    /* preload protection ends at this time */
  int64_t last_use_us;         /* time of the last turn begin or end (LRU order) */
} lv_session_state;

typedef struct lv_event {      /* 32 bytes */
  int32_t kind;                /* LV_EV_* */
  int32_t sid;
  int64_t t_us;
  int64_t a;
  int64_t b;
} lv_event;

typedef struct lv_victim {     /* one block chosen for eviction */
  int32_t sid;
  int32_t blk;
  int32_t page;                /* its HBM page */
} lv_victim;

typedef struct lv_remap_entry {  /* commit block (sid, blk) to location loc (encoded) */
  int32_t sid;
  int32_t blk;
  int32_t loc;
} lv_remap_entry;

typedef struct lv_stats {
  int64_t hbm_allocated;       /* HBM pages reserved or owned */
  int64_t host_allocated;      /* host slots reserved or owned */
  int64_t hbm_budget_pages;
  int64_t host_pages;
  int64_t error;               /* sticky lv_status of the first device-detected error */
  int64_t error_detail;        /* index of the offending item */
  int64_t last_select_count;   /* victims selected by the last ranking (lv_select_victims or a
                                  device-driven step's; 0 for a step with no deficit) */
  int64_t last_select_total;   /* candidate blocks the last ranking that ran saw (a device-driven
                                  step with no deficit ranks nothing and leaves it as it was) */
  /* counters of policy fallbacks and of preload outcomes (Section 6) */
  int64_t selects, victims, shortfalls, pages_out, pages_in, bytes_out, bytes_in;
  int64_t remap_entries, appended_pages, cancels, events, fallback_selects;
  int64_t preloads, preloads_skipped;   /* lv_make_resident with LV_RESIDENT_PRELOAD */
  /* LV_TIERS_INCLUSIVE: clean copies held now (part of host_allocated), evictions
     that found one and moved no bytes (part of pages_out, not of bytes_out), and
     copies dropped because their block gained rows */
  int64_t clean_copies, clean_out, clean_dropped;
} lv_stats;

/* ---------------------------------------------------------------- pool */

/* Section 6 ("Hierarchical KV cache manager"): the paged block pool with side
   tables.  Validates the descriptor, allocates the device metadata (session
   table, block tables, owner tables, allocation bitmaps, error word and
   counters) and, when desc->host_kv is NULL, a mapped page-locked host pool.
   All tables start empty.  Returns LV_ERR_INVALID for a bad descriptor (sizes
   out of range, P not a multiple of 16, a misaligned or non-device KV pointer,
   a host_kv that is not page-locked), LV_ERR_OOM or LV_ERR_CUDA.
   Launch shapes can be overridden through the environment at creation time (for
   tuning sweeps): LV_EXCHANGE_CTAS (the exchange copy's grid, default 3/10 of
   the SMs) or LV_EXCHANGE_CTAS_PER_SM; LV_STAGE_STAGES and LV_STAGE_CTAS_PER_SM
   (the TMA pack/unpack kernel, default about 48 KiB of stages per CTA and two
   CTAs per SM); LV_STAGE_KERNEL=lsu (16-byte copies instead of TMA);
   LV_REMAP_ENTRIES_PER_THREAD = 1, 2 or 4 (lv_remap's entries per thread,
   default 1 while the GPU holds one thread per entry at once, else 2 or 4);
   LV_EXCHANGE_KERNEL=tma (the exchange copy by TMA bulk copies, one issuing
   thread per CTA, with LV_EXCHANGE_STAGES stages of 2P bytes, default 4);
   LV_STEP_GRAPHS=0 (a device-driven step whose kernels all run on the caller's
   stream is issued kernel by kernel instead of as one CUDA graph launch; the
   results are the same). */
lv_status lv_pool_create(const lv_pool_desc* desc, lv_stream stream, lv_pool** out);

/* Waits for the pool's outstanding work on `stream`, then frees everything the
   library allocated.  The caller's KV arrays and host pool are not touched. */
lv_status lv_pool_destroy(lv_pool* pool, lv_stream stream);

/* Host-visible address of the host pool ([host_pages][2L][P]). */
void* lv_pool_host_ptr(lv_pool* pool);

/* Device-visible address of the same host pool (kernels may read and write it
   over the host link; on GB300 it equals the host address). */
void* lv_pool_host_device_ptr(lv_pool* pool);

/* Loads a placement: placement is int32 [max_sessions][max_blocks] of encoded
   entries, ctx_tokens is int32 [max_sessions].  Block b of session s must be
   placed (entry != -1) exactly when b < ceil(ctx_tokens[s] / T).  Rebuilds the
   owner tables, bitmaps and counts.  Device-detected: LV_ERR_DOUBLE_MAP (two
   blocks on one location), LV_ERR_BOUNDS, LV_ERR_BUDGET. */
lv_status lv_pool_import(lv_pool* pool, const int32_t* placement, const int32_t* ctx_tokens,
                         lv_stream stream);

/* ------------------------------------------------------------ sessions */

/* Writes states[0..n) to sessions first..first+n (ctx_tokens is ignored).
   LV_ERR_INVALID when [first, first+n) is not within 0..max_sessions. */
lv_status lv_session_set(lv_pool* pool, const lv_session_state* states, int32_t first,
                         int32_t n, lv_stream stream);

/* Reads sessions first..first+n into out (host or device).  LV_ERR_INVALID
   when [first, first+n) is not within 0..max_sessions. */
lv_status lv_session_get(lv_pool* pool, lv_session_state* out, int32_t first, int32_t n,
                         lv_stream stream);

/* Section 3 (runtime monitor: playback position, user speech, barge-in)
   and Sections 5.1-5.2: applies n events in order to the session table.
   TURN_BEGIN sets RUNNING, clears IMMEDIATE and the preload protection.
   TURN_END(a, b) clears RUNNING, starts a reply of a us and b units (LV_RESP_OPEN).
   Both set last_use_us = t.
   PLAYBACK(a) advances play_us by a, at most to gen_us; reaching it ends the
   reply and records t_done_us.  SPEECH_START sets IMMEDIATE.  BARGE_IN sets
   gen_us = play_us (unplayed audio discarded), ends the reply without a
   completion time, sets IMMEDIATE.  SPEECH_STOP clears IMMEDIATE and, when the
   reply had completed, folds x = t - t_done_us into the reply-interval average
   (first sample: ema = x; later: ema = floor((3*ema + x) / 4)).  PRELOADED
   sets protect_until_us = t + protect_us; UNPROTECT sets it to 0.  Device-detected: LV_ERR_BOUNDS for an
   unknown kind or session id (that event is skipped). */
lv_status lv_session_events(lv_pool* pool, const lv_event* events, int64_t n, lv_stream stream);

/* Section 5.1 / Eq. 4 and "Eviction policy": ranks every HBM-resident block of
   every candidate session by (T_next descending, session id ascending, block
   id descending -- suffix first; ascending under LV_ASCENDING) and writes the
   first min(k, capacity, #candidates) to out (lv_victim [capacity]).
   T_next = T_play + T_reply, clamped to [0, 2^32-1]: T_play = max(0, gen - play)
   (or reply_tokens * unit_us while the reply is open, in LV_PLAY_COUNTERS mode),
   T_reply = reply_ema_us if reply_n > 0 else reply_prior_us.  Candidates are
   sessions that are neither RUNNING nor IMMEDIATE nor protected
   (now_us < protect_until_us).  With LV_SELECT_FALLBACK, protected sessions
   that are not RUNNING follow as a second tier, in the same order.  The count
   written goes to *count_out (int64, host or device; may be NULL); fewer than k
   candidates is not an error (the count says so) and is counted as a shortfall. */
lv_status lv_select_victims(lv_pool* pool, int64_t now_us, int64_t k, uint32_t flags,
                            lv_victim* out, int64_t capacity, int64_t* count_out,
                            lv_stream stream);

/* ------------------------------------------------------------ movement */

/* Section 5 (Fig. 6, eviction to DRAM) / Section 6 (offload connector):
   reserves the n lowest-numbered free host slots (ascending, in victim order)
   and copies every sub-page of each victim's HBM page into its slot.  Does not
   change the block tables: the victims stay valid until lv_remap commits.
   slots_out (int32 [n], may be NULL) receives the slots, commit_out
   (lv_remap_entry [n], may be NULL) ready-to-commit entries.  mode:
   LV_MODE_ZERO_COPY (SM copies straight into the mapped host pool),
   LV_MODE_STAGED (pack into HBM staging, then copy-engine transfer) or
   LV_MODE_AUTO (zero-copy).  LV_TIERS_INCLUSIVE: a victim that has a clean
   copy gets that slot, reserves nothing and moves no bytes; the others reserve
   the lowest free slots in victim order.  LV_MODE_STAGED reads the reserved slots back
   to build one copy per contiguous slot run, so it waits on the host for the
   work queued before it on `stream` (and for the reservation).  Device-detected: LV_ERR_NO_HOST (nothing reserved or copied),
   LV_ERR_BOUNDS, LV_ERR_STATE (a victim is not resident where it says). */
lv_status lv_swap_out(lv_pool* pool, const lv_victim* victims, int64_t n, int32_t* slots_out,
                      lv_remap_entry* commit_out, int32_t mode, lv_stream stream);

/* Section 5.2 (speech-triggered preload) and the synchronous load of Section 6:
   reserves the n lowest-free HBM pages (ascending, in list order) and copies
   each listed host-resident block of session sid into its page.  Does not
   change the block tables.  pages_out (int32 [n]) and commit_out
   (lv_remap_entry [n]) may be NULL.  A preload is this call on a side stream.
   mode as for lv_swap_out (LV_MODE_STAGED: copy-engine transfer of each
   contiguous slot run into HBM staging, then an unpack kernel; it waits on
   the host for the work queued before it).
   Device-detected: LV_ERR_NO_HBM (budget short: nothing reserved or copied),
   LV_ERR_BOUNDS, LV_ERR_STATE (a block is not in the host tier). */
lv_status lv_swap_in(lv_pool* pool, int32_t sid, const int32_t* blks, int64_t n,
                     int32_t* pages_out, lv_remap_entry* commit_out, int32_t mode,
                     lv_stream stream);

/* Section 5.1 (evict until enough HBM is free) followed by the load of
   Section 5.2 / Section 6, as one step: evicts n_out victims to the host tier
   and loads n_in host-resident blocks of session sid, committing both.  The
   result -- slots_out (int32 [n_out], victim order), pages_out (int32 [n_in],
   list order), block and owner tables, bitmaps, counters, bytes -- is exactly
   that of lv_swap_out, lv_remap (its commits), lv_swap_in, lv_remap (its
   commits) issued one after the other: victims take the lowest free host
   slots before any slot is freed, incoming blocks take the lowest free HBM
   pages after the victims' pages are freed.  All metadata is decided first by
   one small kernel; then one copy kernel moves both directions together (an
   incoming block that lands on a victim's old page is copied by the same
   thread right after it read the old bytes), so the host link carries data
   both ways at once.  LV_MODE_STAGED instead packs the evicted pages into HBM
   staging and unpacks the loaded ones, with the copy engines carrying one
   transfer per contiguous slot run in each direction on two side streams (it
   waits on the host for the plan).  Either list may be empty.  The whole call is validated
   before anything changes: on LV_ERR_STATE / LV_ERR_BOUNDS (a victim not
   resident where it says, a block not in the host tier, a block listed twice),
   LV_ERR_NO_HOST or LV_ERR_NO_HBM (device-detected) nothing is reserved,
   committed or copied, and the outputs are -1. */
lv_status lv_swap_exchange(lv_pool* pool, const lv_victim* victims, int64_t n_out, int32_t sid,
                           const int32_t* blks, int64_t n_in, int32_t* slots_out,
                           int32_t* pages_out, int32_t mode, lv_stream stream);

/* lv_make_resident flags and result.  LV_RESIDENT_ASYNC_COPY (lv_make_resident,
   lv_turn): the step's page copies run on the pool's own copy stream, after the
   step's decisions and after every earlier asynchronous copy, so that the work
   queued next on `stream` (the next step's ranking and planning) overlaps
   them.  Until lv_join(pool, stream) the moved KV bytes must not be read or
   written by the caller; every liblv call that moves or reads KV bytes, and
   lv_sync, joins first by itself. */
enum { LV_RESIDENT_PRELOAD = 1, LV_RESIDENT_ASYNC_COPY = 2 };
enum { LV_RESIDENT_DONE = 0, LV_RESIDENT_SKIPPED = 1, LV_RESIDENT_NOTHING = 2,
       LV_RESIDENT_FAILED = 3 /* a device-detected error stopped it (see lv_sync) */ };

typedef struct lv_resident_result {
  int64_t k;              /* pages the HBM budget was short (victims asked for) */
  int64_t n_found;        /* victims the ranking found (min(k, candidates)) */
  int64_t n_victims;      /* victims evicted */
  int64_t n_loaded;       /* host blocks loaded */
  int64_t n_appended;     /* new pages for appended tokens */
  int32_t status;         /* LV_RESIDENT_DONE / _SKIPPED / _NOTHING */
  int32_t sid;            /* the session made resident (lv_turn: the one it picked) */
} lv_resident_result;

/* Sections 5.1 and 5.2, one step with no host round trip: makes session sid
   fully resident and grows its context by append_tokens.  On the device, in
   stream order: list sid's host-tier blocks (ascending); k = max(0, host
   blocks + new blocks - free budget); rank with lv_select_victims' order and
   take the first k (with LV_SELECT_FALLBACK unless LV_RESIDENT_PRELOAD);
   then evict and load exactly as lv_swap_exchange does; then append as
   lv_session_append does.  The results equal those of the host-driven
   sequence select -> exchange -> append.
   Foreground (flags 0): fewer than k victims is LV_ERR_NO_HBM (device-
   detected) and nothing moves.  Preload (LV_RESIDENT_PRELOAD, Section 5.2):
   no host blocks gives LV_RESIDENT_NOTHING; more than max_load_pages host
   blocks (admission; < 0 means no limit) or fewer than k victims gives
   LV_RESIDENT_SKIPPED and nothing moves; a completed preload protects the
   session until now_us + protect_us.  append_tokens must be 0 for a preload.
   Optional outputs (host or device, NULL to skip): victims_out
   (lv_victim [hbm_budget_pages]), slots_out (int32 [hbm_budget_pages]),
   blocks_out and pages_out (int32 [max_blocks]: blocks loaded and their
   pages), append_out (int32 [append_tokens / T + 2]), result_out. */
lv_status lv_make_resident(lv_pool* pool, int32_t sid, int64_t now_us, int32_t append_tokens,
                           uint32_t flags, int64_t max_load_pages, lv_victim* victims_out,
                           int32_t* slots_out, int32_t* blocks_out, int32_t* pages_out,
                           int32_t* append_out, lv_resident_result* result_out,
                           lv_stream stream);

/* Section 6 (side tables) and Section 5.2 (a failed
   preload costs time, never correctness): commits n entries.  For each, the new location must be a
   reservation not yet owned; it becomes owned by (sid, blk), the block table
   points to it and the old location is freed.  LV_TIERS_INCLUSIVE: a host
   location may also be the block's own clean copy (it then stops being a
   copy); a block committed to HBM from the host tier keeps its slot as its
   clean copy; a block committed to another host slot loses its clean copy
   (freed).  Entries are independent;
   a bad one is skipped.  Device-detected: LV_ERR_DOUBLE_MAP (location not a
   free reservation, or the same block twice in one call), LV_ERR_BOUNDS,
   LV_ERR_BUDGET. */
lv_status lv_remap(lv_pool* pool, const lv_remap_entry* entries, int64_t n, lv_stream stream);

/* Releases reservations that will never be committed (a cancelled or failed
   transfer, Section 5.2).  locs are encoded locations.  A host slot that is
   its owner's clean copy (LV_TIERS_INCLUSIVE) was not reserved and is left as
   it is.  Device-detected: LV_ERR_STATE when a location is owned or not
   reserved. */
lv_status lv_cancel(lv_pool* pool, const int32_t* locs, int64_t n, lv_stream stream);

/* Section 5.1 under memory pressure from outside the manager, with no host
   round trip: frees up to k HBM pages now.  On the device, in stream order:
   rank with lv_select_victims' order (normal eligibility, no fallback tier),
   take the first k -- every candidate when there are fewer -- and evict them
   exactly as lv_swap_exchange does with no incoming blocks.  The results
   equal those of lv_select_victims followed by lv_swap_exchange.
   flags: 0 or LV_RESIDENT_ASYNC_COPY.  Optional outputs (host or device, NULL
   to skip): victims_out (lv_victim [hbm_budget_pages]: the victims chosen),
   slots_out (int32 [hbm_budget_pages]: their host slots), result_out (k, and
   n_found = n_victims = victims evicted; n_loaded = 0; status
   LV_RESIDENT_DONE, or LV_RESIDENT_NOTHING when nothing was a candidate;
   sid = -1).  k above hbm_budget_pages is taken as hbm_budget_pages.
   Device-detected: LV_ERR_NO_HOST when the host tier cannot take the victims
   (then nothing moves). */
lv_status lv_evict(lv_pool* pool, int64_t now_us, int64_t k, uint32_t flags, lv_victim* victims_out,
                   int32_t* slots_out, lv_resident_result* result_out, lv_stream stream);

/* One turn of a voice session as one call (Section 3: the user's input is
   complete and the request runs; Sections 5.1 and 5.2: its KV is made
   resident first), with no host round trip.  In stream order on the device:
   the turn's session is d->sid, or, when d->sid is -1, the first of
   d->candidates (num_candidates session ids, device or host memory, read at
   call time) that has at least one block in the host tier -- the first
   candidate when none has; then LV_EV_TURN_BEGIN at now_us; then
   lv_make_resident(sid, now_us, append_tokens, foreground); then, unless that
   failed, LV_EV_TURN_END at now_us with a = reply_audio_us, b = reply_units.
   The outputs are those of lv_make_resident (each may be NULL), with
   result.sid the session.  load_keys (optional, uint64 [max_blocks], device
   or host memory, indexed by block id) sets the order in which the session's
   host-tier blocks are loaded -- ascending (key, block id) instead of
   ascending block id -- and so which of the lowest free HBM pages each block
   takes; blocks_out then lists them in that order.  Ordering costs one warp
   per host block, each comparing it with every other.  Host-detected:
   LV_ERR_INVALID.  Device-detected: as lv_make_resident, LV_ERR_BOUNDS for a
   candidate out of range. */
typedef struct lv_turn_desc {
  int32_t sid;                 /* the session, or -1: pick from candidates */
  int32_t num_candidates;      /* 1..max_sessions when sid == -1 */
  const int32_t* candidates;   /* session ids in pick order */
  int64_t now_us;              /* the turn's start */
  int64_t reply_audio_us;      /* LV_EV_TURN_END a: audio of the reply */
  int64_t reply_units;         /* LV_EV_TURN_END b: reply length in progress units */
  int32_t append_tokens;       /* context growth (>= 0) */
  uint32_t flags;              /* 0 or LV_RESIDENT_ASYNC_COPY */
  const uint64_t* load_keys;   /* NULL, or the load order's key of every block */
} lv_turn_desc;
lv_status lv_turn(lv_pool* pool, const lv_turn_desc* d, lv_victim* victims_out, int32_t* slots_out,
                  int32_t* blocks_out, int32_t* pages_out, int32_t* append_out,
                  lv_resident_result* result_out, lv_stream stream);

/* Makes `stream` wait for every page copy issued so far with
   LV_RESIDENT_ASYNC_COPY (nothing to wait for: no effect). */
lv_status lv_join(lv_pool* pool, lv_stream stream);

/* The staged path's building blocks (Section 6, offload connector), usable on
   their own: lv_pack_pages gathers the 2L sub-pages of each listed HBM page into
   one contiguous run, dst[i][j] = hbm_kv[j][pages[i]] (dst [n][2L][P]);
   lv_unpack_pages scatters such a run back, hbm_kv[j][pages[i]] = src[i][j].
   The run must be device memory or mapped page-locked host memory, 16-byte
   aligned.  They move raw bytes and touch no table: the caller decides which
   pages may be read or written.  Device-detected: LV_ERR_BOUNDS for a page id
   outside the pool (that page is skipped). */
lv_status lv_pack_pages(lv_pool* pool, const int32_t* pages, int64_t n, void* dst, lv_stream stream);
lv_status lv_unpack_pages(lv_pool* pool, const void* src, const int32_t* pages, int64_t n,
                          lv_stream stream);

/* Reads listed HBM pages and reduces each to a 64-bit checksum: with the
   page's 2L sub-pages concatenated in order (sub-page j = 2*layer + kv) and
   read as little-endian 64-bit words w_0 .. w_{m-1} (m = 2L*P/8),
       sums_out[i] = sum over q of w_q * (2q + 1)   (mod 2^64).
   The weights make the sum depend on where each word sits.  It stands in for
   a consumer that reads running sessions' KV (attention reads every byte of
   a page) and verifies page contents without copying them to the host.  Not
   from the paper: an instrument.  sums_out (uint64 [n], device or host).
   Device-detected: LV_ERR_BOUNDS for a page outside the pool (its sum is 0). */
lv_status lv_page_checksums(lv_pool* pool, const int32_t* pages, int64_t n, uint64_t* sums_out,
                            lv_stream stream);

/* Block-level allocation kept (Section 5.1): grows session sid's context by
   n_tokens; each new block takes the lowest free HBM page, in block order, and
   is committed at once.  LV_TIERS_INCLUSIVE: when n_tokens > 0 and the last
   block is partially filled, its clean copy (if any) is dropped.  pages_out (int32, capacity ceil(n_tokens/T)+1, may be
   NULL) receives the new pages; *count_out (int32, may be NULL) their number.
   Device-detected: LV_ERR_NO_HBM (nothing changes), LV_ERR_BOUNDS (the block
   table would overflow). */
lv_status lv_session_append(lv_pool* pool, int32_t sid, int32_t n_tokens, int32_t* pages_out,
                            int32_t* count_out, lv_stream stream);

/* --------------------------------------------------------------- views */

/* Per-session counts of blocks in HBM and in the host tier (int32 [S] each,
   either may be NULL). */
lv_status lv_session_counts(lv_pool* pool, int32_t* hbm_blocks, int32_t* host_blocks,
                            lv_stream stream);

/* The blocks of session sid in one tier (where 0: HBM, 1: host), ascending,
   into blks_out (int32, capacity max_blocks); *count_out (int64) their number. */
lv_status lv_session_blocks(lv_pool* pool, int32_t sid, int32_t where, int32_t* blks_out,
                            int64_t* count_out, lv_stream stream);

/* Copies the block tables (int32 [S][max_blocks]) and, if not NULL, the owner
   tables (int32 [hbm_pages] and [host_pages]: sid << 16 | blk for an owned
   location, -1 free, -2 reserved by a swap and not yet committed). */
lv_status lv_read_tables(lv_pool* pool, int32_t* tables, int32_t* hbm_owner,
                         int32_t* host_owner, lv_stream stream);

/* ------------------------------------------- ranking without allocation */

/* The paper has no counterpart to this entry point; it exists for callers of
   this library that must not allocate GPU memory while they rank victims -- an
   engine that has already given nearly all free HBM to its KV pages, where a
   further cudaMalloc can fail or fragment that reservation, or a
   latency-critical scheduler thread, where cudaMalloc / cudaFree can
   synchronise the device.

   lv_select_victims_noalloc computes what lv_select_victims computes on a pool
   of the same policy, within order and T_play mode (same order, same count,
   same fallback tier), but from a session table and block tables that the
   caller passes in, without a pool: sessions is lv_session_state
   [num_sessions] (ctx_tokens gives each session's block count), tables is
   int32 [num_sessions][max_blocks] in the block-table encoding above.  Both,
   and out (lv_victim [capacity]) and count_out (int64, may be NULL), must be
   memory that the current device can address: device memory of the current
   device, managed memory, or mapped page-locked host memory with a device
   alias for it.  Pageable host pointers (staging them would need an
   allocation) and device memory of another device are rejected with
   LV_ERR_INVALID.

   Its working memory is one array of LV_NOALLOC_MAX_SESSIONS x 20 bytes plus
   256 bytes (80.25 KiB) compiled into liblv as device memory: every GPU that
   loads the library holds it until the process exits.  num_sessions above
   LV_NOALLOC_MAX_SESSIONS is rejected with LV_ERR_INVALID.  The call issues no
   cudaMalloc, cudaFree or allocating library routine.  The first call on a
   device looks up that array's device address (cudaGetSymbolAddress) and
   keeps it for the rest of the process, so make the first call on each device
   before any stream capture; under lazy module loading (the CUDA default) that
   first call, or the first ranking of any kind on the device, may also load
   liblv's kernels, which takes device memory once.  A warm-up call at
   start-up, before the memory is given away, leaves every later call free of
   allocations.  The kept address does not survive cudaDeviceReset or the
   destruction of the device's primary context: do not call it after either.
   All calls on a device share the one array and each call starts by clearing
   its counters: calls whose execution overlaps on the GPU (two streams, or two
   host threads) race and may return wrong victims, so order them, for example
   on one stream. */
#define LV_NOALLOC_MAX_SESSIONS 4096

typedef struct lv_rank_params {
  int32_t num_sessions;        /* 1..LV_NOALLOC_MAX_SESSIONS */
  int32_t max_blocks;          /* row length of the block tables, 1..65536 */
  int32_t page_tokens;         /* T */
  int32_t within_order;        /* LV_SUFFIX_FIRST or LV_ASCENDING */
  int32_t t_play_mode;         /* LV_PLAY_PLAYBACK or LV_PLAY_COUNTERS */
  uint32_t flags;              /* 0 or LV_SELECT_FALLBACK */
  int64_t reply_prior_us;      /* >= 0 */
  int64_t unit_us;             /* 1..2^31 */
  int32_t policy;              /* LV_POLICY_NEXT_USE or LV_POLICY_LRU */
  int32_t reserved;            /* must be 0 */
} lv_rank_params;

lv_status lv_select_victims_noalloc(const lv_rank_params* params, const lv_session_state* sessions,
                                    const int32_t* tables, int64_t now_us, int64_t k,
                                    lv_victim* out, int64_t capacity, int64_t* count_out,
                                    lv_stream stream);

/* --------------------------------------------------- request scheduling */

/* One ready request of a stage for lv_schedule (48 bytes). */
typedef struct lv_request {
  int32_t id;                  /* caller's request id (echoed in the order) */
  int32_t started;             /* 1 once its first playable audio went out */
  int64_t play_buffer_us;      /* P_i: audio the client holds, 0..2^40 */
  int64_t ready_age_us;        /* A_i: time since it became ready, 0..2^62 */
  int64_t kv_pages;            /* K_i: GPU KV it occupies, 0..2^24 pages */
  int64_t tokens;              /* token budget it consumes if admitted (>= 0) */
  int64_t kv_needed;           /* KV blocks it needs if admitted (>= 0) */
} lv_request;

typedef struct lv_sched_params {
  int64_t p_safe_us;           /* P_safe, 1..2^32 */
  int64_t alpha, beta;         /* Eq. 1 weights, 0..2^16 */
  int64_t occupied;            /* occupied GPU KV of the stage, 0..2^32 */
  int64_t allocatable;         /* allocatable GPU KV of the stage, 1..2^32 */
  int64_t token_budget;        /* round budgets M_s */
  int64_t kv_budget;
} lv_sched_params;

#define LV_SCHED_MAX_REQUESTS 4096

/* Section 4.1 (urgency classes, Eqs. 1-3) and Section 4.2 (Algorithm 1): one
   scheduling round over n ready requests (reqs, lv_request [n]).  Class U0
   (started, P_i <= P_safe) by P_i ascending; U1 (not started) by A_i
   descending; U2 (started, P_i > P_safe) by U_i = beta*K_i*R_occ -
   alpha*max(0, P_i - P_safe)/P_safe descending, R_occ = occupied/allocatable;
   ties keep the ready set's order.  order_out (int32 [n]) receives the request
   ids in priority order U0-U1-U2; *batch_out (int32) the length of the
   admitted prefix: admission stops at the first request whose tokens or KV
   blocks exceed what is left of the round budgets.  Exact integer arithmetic;
   the pool's scheduling scratch (128 KiB), so calls on one pool are ordered on
   one stream.  n is 0..LV_SCHED_MAX_REQUESTS.  Device-detected:
   LV_ERR_BOUNDS for a field outside its range (it is clamped). */
lv_status lv_schedule(lv_pool* pool, const lv_sched_params* params, const lv_request* reqs, int32_t n,
                      int32_t* order_out, int32_t* batch_out, lv_stream stream);

/* ------------------------------------------------------------- status */

/* Synchronous: waits for `stream`, returns the sticky device error (LV_OK if
   none) or LV_ERR_CUDA. */
lv_status lv_sync(lv_pool* pool, lv_stream stream);

/* Synchronous: waits for `stream` and fills *out. */
lv_status lv_get_stats(lv_pool* pool, lv_stats* out, lv_stream stream);

/* Clears the sticky device error (stream-ordered). */
lv_status lv_clear_error(lv_pool* pool, lv_stream stream);

/* Instrumentation (Section 6: counters that validate which paths run).  While
   enabled, every launch of a copy kernel -- swap-out, swap-in, exchange, and the
   staged path's pack and unpack -- is bracketed by two CUDA events recorded on
   its own stream.  lv_timing_read waits for them and reports, per kernel kind
   (index LV_TIMING_*), the launches and their summed, shortest and longest
   durations; reset != 0 starts a new record.  Enabling it adds two event
   records per launch and nothing else. */
enum { LV_TIMING_SWAP_OUT = 0, LV_TIMING_SWAP_IN = 1, LV_TIMING_EXCHANGE = 2, LV_TIMING_PACK = 3,
       LV_TIMING_UNPACK = 4, LV_TIMING_KINDS = 5 };
typedef struct lv_kernel_timing {
  int64_t launches;
  double total_ms;
  double min_ms;
  double max_ms;
} lv_kernel_timing;
lv_status lv_timing_enable(lv_pool* pool, int32_t enable);
lv_status lv_timing_read(lv_pool* pool, lv_kernel_timing* out /* [LV_TIMING_KINDS] */, int32_t reset);

/* Failure paths without a GPU fault (Section 5.2: a failed or cancelled
   transfer must leave the old mapping valid).  lv_inject_fault arms a one-shot
   fault: the (after+1)-th later host-slot allocation (LV_FAULT_HOST_ALLOC) or
   HBM-page allocation (LV_FAULT_HBM_ALLOC) fails as if that tier were full --
   the device reports LV_ERR_NO_HOST / LV_ERR_NO_HBM and nothing is reserved or
   copied -- or the (after+1)-th later copy-engine transfer of the staged path
   (LV_FAULT_COPY) is not issued and the call returns LV_ERR_CUDA, leaving the
   reservations made so far uncommitted (release them with lv_cancel).
   LV_FAULT_NONE disarms.  lv_selftest_wait runs the library's bounded device
   wait on a barrier that nothing completes, with a limit of limit_us; the
   device then reports LV_ERR_TIMEOUT and the context stays usable. */
enum { LV_FAULT_NONE = 0, LV_FAULT_HOST_ALLOC = 1, LV_FAULT_HBM_ALLOC = 2, LV_FAULT_COPY = 3 };
lv_status lv_inject_fault(lv_pool* pool, int32_t kind, int32_t after);
lv_status lv_selftest_wait(lv_pool* pool, int64_t limit_us, lv_stream stream);

/* ------------------------------------------------------ preload controller */

/* Section 5.2, the preload controller, over the pool's own calls.  Readings (the
   paper describes it in prose):
   - Admission: a preload of B bytes requested at time t is admitted if, queued
     behind the transfers already on a modelled host->device link of
     link_bytes_per_us, it finishes by the predicted start of the session's turn,
     t_speech + lead (lead: the session's moving average of turn start minus
     speech start, integer EMA of weight 1/4, first sample sets it; lead_prior_us
     before any sample; t_speech is the first speech start or barge-in since the
     session's last turn), and if the pages it must evict fit in the host tier with
     max_blocks slots still free.
   - A refused preload waits and is re-checked at every later tick until it is
     admitted, its deadline passes (given up), or the turn begins (given up).
   - An admitted preload evicts what it needs (the ranked order, no fallback tier)
     and commits that at once; it reserves and fills its HBM pages at once but
     commits them only at the first tick at or after its modelled finish.  A turn
     that begins first cancels the reservation (the turn then loads itself).
   - A completed preload protects the session until finish + protect_us; when the
     protected sessions' resident pages exceed cap_pages, the oldest protections
     (earliest end, then lower session id) are dropped.
   - A turn's own synchronous load occupies the modelled link too
     (lv_controller_turn_loaded).
   The hooks are called in event order: lv_controller_tick at every event, then
   lv_controller_turn_begin before a turn, lv_controller_speech at a speech start
   or barge-in.  Each hook waits on the host for the work queued before it on
   `stream` (it reads host blocks, allocation counts and session states). */
typedef struct lv_controller lv_controller;
typedef struct lv_controller_desc {
  int64_t link_bytes_per_us;   /* > 0 */
  int64_t lead_prior_us;       /* >= 0 */
  int64_t cap_pages;           /* resident pages of protected sessions at most; -1: no cap */
  int32_t mode;                /* LV_MODE_* of the preloads' and evictions' copies */
  int32_t reserved;            /* must be 0 */
} lv_controller_desc;
/* decision records, in the order the decisions were taken */
enum { LV_CTL_ADMITTED = 1, LV_CTL_COMPLETED = 2, LV_CTL_CANCELLED = 3, LV_CTL_GIVEN_UP = 4,
       LV_CTL_UNPROTECTED = 5, LV_CTL_EVICTED = 6 };
typedef struct lv_controller_record {
  int32_t kind;                /* LV_CTL_* */
  int32_t sid;                 /* the session (EVICTED: the session being preloaded) */
  int64_t start_us, finish_us, deadline_us;   /* ADMITTED: the modelled transfer */
  int64_t n;                   /* ADMITTED: pages loaded; EVICTED: victims */
  int64_t data_offset;         /* ADMITTED: n HBM pages; EVICTED: n (sid, blk, page) triples */
} lv_controller_record;
typedef struct lv_controller_counters {
  int64_t admitted, completed, waited, given_up, cancelled, hits, victims, pages_in;
} lv_controller_counters;
/* A controller over `pool` (one per pool).  LV_ERR_INVALID for a bad descriptor. */
lv_status lv_controller_create(lv_pool* pool, const lv_controller_desc* d, lv_controller** out);
/* Cancels pending preloads (their reservations are released) and frees the
   controller; call it before lv_pool_destroy of its pool. */
lv_status lv_controller_destroy(lv_controller* c, lv_stream stream);
lv_status lv_controller_tick(lv_controller* c, int64_t now_us, lv_stream stream);
lv_status lv_controller_speech(lv_controller* c, int32_t sid, int64_t now_us, lv_stream stream);
lv_status lv_controller_turn_begin(lv_controller* c, int32_t sid, int64_t now_us, lv_stream stream);
lv_status lv_controller_turn_loaded(lv_controller* c, int64_t now_us, int64_t pages);
/* Moves the records taken since the last call (and their int32 data) to the caller.
   With too small a capacity nothing moves, *n_records and *n_data receive the sizes
   needed, and the call returns LV_ERR_INVALID. */
lv_status lv_controller_records(lv_controller* c, lv_controller_record* records, int64_t capacity,
                                int64_t* n_records, int32_t* data, int64_t data_capacity,
                                int64_t* n_data);
/* The controller's counters since it was created (host memory). */
lv_status lv_controller_counters_get(lv_controller* c, lv_controller_counters* out);

/* A static, human-readable name of a status. */
const char* lv_status_str(lv_status s);
/* The library's interface version: LV_VERSION of the header it was built with.  A
   caller built against another header must not use the library. */
#define LV_VERSION 3
int32_t lv_version(void);

#ifdef __cplusplus
}
#endif
#endif /* LV_H */
