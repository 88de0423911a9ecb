// lv_probe_scattered: an instrument that measures how fast this GPU serves
// scattered 4-byte loads, stores and atomics.
//
// Remap and the other metadata kernels touch one 4-byte word in each 32-byte
// sector they visit, at positions that follow the block tables, so a streaming
// copy is the wrong ceiling for them.  This kernel issues the same kind of
// traffic with nothing else in it: every thread makes a given mix of loads,
// returning atomics, stores and reductions at hashed positions in a
// caller-owned array.  The caller times the launch: one kind alone gives the
// rate at which the GPU serves that kind, and a kernel's own mix per work item
// with one thread per item gives that kernel's ceiling.
#include <cstdint>

#include "lv_internal.cuh"

namespace {

constexpr int kProbeThreads = 256;
constexpr int kProbeMaxPerKind = 64;

// A 32-bit integer hash (an xor-shift-multiply finaliser); positions only need
// to be spread evenly, not to be unpredictable.
__device__ __forceinline__ uint32_t spread(uint32_t x) {
  x ^= x >> 16;
  x *= 0x7feb352dU;
  x ^= x >> 15;
  x *= 0x846ca68bU;
  x ^= x >> 16;
  return x;
}

// Thread i makes its loads, then its returning atomics, then its stores, then its
// reductions; request r of the thread goes to word spread(i * total + r) & mask.
// No request depends on another, so the GPU may keep all of them in flight.
__global__ void __launch_bounds__(kProbeThreads)
k_probe_scattered(uint32_t* __restrict__ a, uint32_t mask, long long threads, lv_probe_mix m,
                  uint32_t* sink) {
  const long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  if (i >= threads) return;
  const int total = m.loads + m.atomics + m.stores + m.reductions;
  uint32_t r = (uint32_t)i * (uint32_t)total + 0x9e3779b9U;
  uint32_t acc = 0;
#pragma unroll 8
  for (int q = 0; q < m.loads; ++q) acc += a[spread(r++) & mask];
#pragma unroll 8
  for (int q = 0; q < m.atomics; ++q) acc += atomicExch(&a[spread(r++) & mask], (uint32_t)i);
#pragma unroll 8
  for (int q = 0; q < m.stores; ++q) a[spread(r++) & mask] = (uint32_t)i;
#pragma unroll 8
  for (int q = 0; q < m.reductions; ++q) atomicAnd(&a[spread(r++) & mask], 0xFFFFFFF0U);
  // keeps the loads and returned values live; the condition is never met by design
  if (acc == 0x5a5a5a5aU && sink) *sink = acc;
}

}  // namespace

extern "C" lv_status lv_probe_scattered(const lv_probe_mix* mix, uint32_t* array, int64_t words,
                                        int64_t threads, uint32_t* sink, lv_stream stream) {
  if (!mix || !array || words < 1 || (words & (words - 1)) != 0 || words > (1ll << 32))
    return LV_ERR_INVALID;
  if (threads < 1 || threads > (1ll << 31)) return LV_ERR_INVALID;
  const lv_probe_mix m = *mix;
  for (int32_t c : {m.loads, m.atomics, m.stores, m.reductions})
    if (c < 0 || c > kProbeMaxPerKind) return LV_ERR_INVALID;
  const long long grid = (threads + kProbeThreads - 1) / kProbeThreads;
  k_probe_scattered<<<grid, kProbeThreads, 0, static_cast<cudaStream_t>(stream)>>>(
      array, (uint32_t)(words - 1), threads, m, sink);
  return cudaGetLastError() == cudaSuccess ? LV_OK : LV_ERR_CUDA;
}
