// lv_schedule: the interaction-aware request scheduler of Section 4 (Algorithm 1).
//
// A ready set of up to LV_SCHED_MAX_REQUESTS requests: every request gets a
// 128-bit key (urgency class, the class's own order, its position in the ready
// set); then each request counts the smaller keys (its place in the order) and
// sums their token and KV costs, which decides whether it lies in the
// longest prefix that fits the round budgets ("admission stops" at the first
// request that does not fit).  Nothing is sorted; the work spreads over the GPU.
#include <cstdint>

#include "lv_internal.cuh"

namespace lv {
namespace {

using u128 = unsigned __int128;
using i128 = __int128;

constexpr int kKeyThreads = 256;
constexpr int kPerWarp = 2;                                   // requests a warp places
constexpr int kPlaceThreads = 512;
constexpr int kPlaceRequests = kPlaceThreads / 32 * kPerWarp;  // requests a CTA places
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

// Every request's 128-bit key and its two costs (negative costs count as 0).
__global__ void __launch_bounds__(kKeyThreads)
k_sched_keys(lv_sched_params q, const lv_request* __restrict__ reqs, int n, u128* __restrict__ keys,
             longlong2* __restrict__ cost, int32_t* __restrict__ batch, long long* __restrict__ err) {
  // the placement grid may be scheduled once every key CTA has started; it waits
  // for all keys (griddepcontrol.wait) before it reads them
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int i = blockIdx.x * kKeyThreads + threadIdx.x;
  if (i == 0) *batch = 0;
  if (i >= n) return;
  const lv_request& r = reqs[i];
  keys[i] = request_key(r, i, q, err);
  cost[i] = make_longlong2(r.tokens > 0 ? r.tokens : 0, r.kv_needed > 0 ? r.kv_needed : 0);
}

// A CTA places 32 requests: each warp holds kPerWarp of them and its lanes
// stride over the ready set, comparing every key (staged in shared memory) with
// the warp's requests.  Keys are distinct (each holds its request's index), so a
// request's place in the priority order is the number of smaller keys, and the
// tokens and KV admitted before it are the sums of their costs.  Costs are never
// negative, so the requests that fit -- cumulative costs through their own
// within both budgets -- are exactly the prefix that admission reaches before it
// stops.
__global__ void __launch_bounds__(kPlaceThreads)
k_sched_place(lv_sched_params q, const lv_request* __restrict__ reqs, int n,
              const u128* __restrict__ keys, const longlong2* __restrict__ cost,
              int32_t* __restrict__ order, int32_t* __restrict__ batch) {
  asm volatile("griddepcontrol.wait;" ::: "memory");   // every key, cost and the zeroed batch
  extern __shared__ __align__(16) unsigned char smem[];
  u128* sk = reinterpret_cast<u128*>(smem);
  longlong2* sc = reinterpret_cast<longlong2*>(sk + n);
  __shared__ int s_admitted;
  if (threadIdx.x == 0) s_admitted = 0;
  for (int j = threadIdx.x; j < n; j += kPlaceThreads) {
    sk[j] = keys[j];
    sc[j] = cost[j];
  }
  __syncthreads();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int base = blockIdx.x * kPlaceRequests + w * kPerWarp;
  u128 mine[kPerWarp];
  int rank[kPerWarp];
  long long tok[kPerWarp], kv[kPerWarp];
#pragma unroll
  for (int r = 0; r < kPerWarp; ++r) {
    mine[r] = base + r < n ? sk[base + r] : ~(u128)0;
    rank[r] = 0;
    tok[r] = kv[r] = 0;
  }
  for (int j = lane; j < n; j += 32) {
    const u128 k = sk[j];
    const longlong2 c = sc[j];
#pragma unroll
    for (int r = 0; r < kPerWarp; ++r) {
      const long long m = k < mine[r] ? -1ll : 0ll;
      rank[r] -= (int)m;
      tok[r] += c.x & m;
      kv[r] += c.y & m;
    }
  }
#pragma unroll
  for (int r = 0; r < kPerWarp; ++r) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      rank[r] += __shfl_xor_sync(0xffffffffu, rank[r], o);
      tok[r] += __shfl_xor_sync(0xffffffffu, tok[r], o);
      kv[r] += __shfl_xor_sync(0xffffffffu, kv[r], o);
    }
    const int i = base + r;
    if (lane == r && i < n) {
      order[rank[r]] = reqs[i].id;
      if (tok[r] + sc[i].x <= q.token_budget && kv[r] + sc[i].y <= q.kv_budget)
        atomicAdd(&s_admitted, 1);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && s_admitted) atomicAdd(batch, s_admitted);
}

}  // namespace

cudaError_t launch_schedule(const lv_sched_params& q, const lv_request* reqs, int n, int32_t* order,
                            int32_t* batch, long long* ctl, void* scratch, cudaStream_t s) {
  u128* keys = static_cast<u128*>(scratch);
  longlong2* cost = reinterpret_cast<longlong2*>(keys + LV_SCHED_MAX_REQUESTS);
  // every CTA stages all keys and costs: 32 B per request, up to 128 KiB
  cudaError_t e = cudaFuncSetAttribute(k_sched_place, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)(32 * LV_SCHED_MAX_REQUESTS));
  if (e != cudaSuccess) return e;
  k_sched_keys<<<(n + kKeyThreads - 1) / kKeyThreads, kKeyThreads, 0, s>>>(q, reqs, n, keys, cost,
                                                                          batch, ctl);
  // programmatic dependent launch: the placement grid's launch overlaps the keys
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)((n + kPlaceRequests - 1) / kPlaceRequests));
  cfg.blockDim = dim3(kPlaceThreads);
  cfg.dynamicSmemBytes = (size_t)n * 32;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, k_sched_place, q, reqs, n, (const u128*)keys, (const longlong2*)cost,
                         order, batch);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace lv
