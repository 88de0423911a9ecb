// lv_schedule: the interaction-aware request scheduler of Section 4 (Algorithm 1).
//
// One CTA ranks a ready set of up to LV_SCHED_MAX_REQUESTS requests: every request
// gets a 128-bit key (urgency class, the class's own order, its position in the
// ready set), a bitonic sort orders the keys in shared memory, and a scan of the
// token and KV costs in that order finds the longest prefix that fits the round
// budgets ("admission stops" at the first request that does not fit).
#include <cstdint>

#include "lv_internal.cuh"

namespace lv {
namespace {

using u128 = unsigned __int128;
using i128 = __int128;

constexpr int kSchedThreads = 1024;
constexpr u128 kLow114 = (((u128)1) << 114) - 1;

__device__ __forceinline__ void sched_error(long long* ctl, int code) {
  atomicCAS(reinterpret_cast<unsigned long long*>(&ctl[C_ERR]), 0ull, (unsigned long long)code);
}

// Class-ordered key, smallest first: class 0 by playback buffer ascending,
// class 1 by ready age descending, class 2 by the Eq. 1 utility descending
// (U scaled by allocatable * P_safe, an exact integer with the same order).
__device__ u128 request_key(const lv_request& r, int idx, const lv_sched_params& q, long long* err) {
  long long P = r.play_buffer_us, A = r.ready_age_us, K = r.kv_pages;
  if (P < 0 || P > (1ll << 40) || A < 0 || A > (1ll << 62) || K < 0 || K > (1ll << 24) ||
      r.tokens < 0 || r.kv_needed < 0) {
    sched_error(err, LV_ERR_BOUNDS);
    P = P < 0 ? 0 : (P > (1ll << 40) ? (1ll << 40) : P);
    A = A < 0 ? 0 : (A > (1ll << 62) ? (1ll << 62) : A);
    K = K < 0 ? 0 : (K > (1ll << 24) ? (1ll << 24) : K);
  }
  unsigned cls;
  u128 v;
  if (!r.started) {
    cls = 1;
    v = (u128)((1ll << 62) - A);
  } else if (P <= q.p_safe_us) {
    cls = 0;
    v = (u128)P;
  } else {
    cls = 2;
    // U' = beta*K*occupied*P_safe - alpha*(P - P_safe)*allocatable, |U'| < 2^105
    const i128 gain = (i128)q.beta * K * q.occupied * q.p_safe_us;
    const i128 cost = (i128)q.alpha * (P - q.p_safe_us) * q.allocatable;
    v = (u128)((((i128)1) << 110) - (gain - cost));
  }
  return ((u128)cls << 126) | ((v & kLow114) << 12) | (u128)(unsigned)idx;
}

__global__ void __launch_bounds__(kSchedThreads)
k_schedule(lv_sched_params q, const lv_request* __restrict__ reqs, int n, int N,
           int32_t* __restrict__ order, int32_t* __restrict__ batch, long long* __restrict__ err) {
  extern __shared__ __align__(16) unsigned char smem[];
  u128* keys = reinterpret_cast<u128*>(smem);
  for (int i = threadIdx.x; i < N; i += kSchedThreads)
    keys[i] = i < n ? request_key(reqs[i], i, q, err) : ~(u128)0;
  __syncthreads();
  for (int k = 2; k <= N; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < N; i += kSchedThreads) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const u128 a = keys[i], b = keys[ixj];
          if (((i & k) == 0) ? (a > b) : (a < b)) {
            keys[i] = b;
            keys[ixj] = a;
          }
        }
      }
      __syncthreads();
    }
  }
  // cumulative token and KV costs in priority order; the admitted set is a prefix
  const int per = (N + kSchedThreads - 1) / kSchedThreads;
  const int r0 = min(N, (int)threadIdx.x * per), r1 = min(N, r0 + per);
  long long tok = 0, kv = 0;
  for (int r = r0; r < r1 && r < n; ++r) {
    const lv_request& x = reqs[(int)(keys[r] & 0xFFF)];
    tok += x.tokens > 0 ? x.tokens : 0;
    kv += x.kv_needed > 0 ? x.kv_needed : 0;
  }
  __shared__ long long s_tok[kSchedThreads], s_kv[kSchedThreads];
  __shared__ int s_cnt[kSchedThreads];
  s_tok[threadIdx.x] = tok;
  s_kv[threadIdx.x] = kv;
  __syncthreads();
  // exclusive prefix over threads (a simple two-array Hillis-Steele scan)
  for (int off = 1; off < kSchedThreads; off <<= 1) {
    const long long at = threadIdx.x >= off ? s_tok[threadIdx.x - off] : 0;
    const long long ak = threadIdx.x >= off ? s_kv[threadIdx.x - off] : 0;
    __syncthreads();
    s_tok[threadIdx.x] += at;
    s_kv[threadIdx.x] += ak;
    __syncthreads();
  }
  long long ctok = s_tok[threadIdx.x] - tok, ckv = s_kv[threadIdx.x] - kv;
  int admitted = 0;
  for (int r = r0; r < r1 && r < n; ++r) {
    const int idx = (int)(keys[r] & 0xFFF);
    const lv_request& x = reqs[idx];
    order[r] = x.id;
    ctok += x.tokens > 0 ? x.tokens : 0;
    ckv += x.kv_needed > 0 ? x.kv_needed : 0;
    admitted += (ctok <= q.token_budget && ckv <= q.kv_budget) ? 1 : 0;
  }
  s_cnt[threadIdx.x] = admitted;
  __syncthreads();
  for (int off = kSchedThreads / 2; off > 0; off >>= 1) {
    if (threadIdx.x < off) s_cnt[threadIdx.x] += s_cnt[threadIdx.x + off];
    __syncthreads();
  }
  if (threadIdx.x == 0) *batch = s_cnt[0];
}

}  // namespace

cudaError_t launch_schedule(const lv_sched_params& q, const lv_request* reqs, int n, int32_t* order,
                            int32_t* batch, long long* ctl, cudaStream_t s) {
  int N = 1;
  while (N < n) N <<= 1;
  const size_t smem = (size_t)N * sizeof(u128);
  cudaError_t e = cudaFuncSetAttribute(k_schedule, cudaFuncAttributeMaxDynamicSharedMemorySize, 64 * 1024);
  if (e != cudaSuccess) return e;
  k_schedule<<<1, kSchedThreads, smem, s>>>(q, reqs, n, N, order, batch, ctl);
  return cudaGetLastError();
}

}  // namespace lv
