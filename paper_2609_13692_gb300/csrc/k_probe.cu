// Measurement helpers, not part of the method.
//
// mpt_gather_bandwidth: the random-gather bandwidth that bounds the naive
// form of the Sec. 3.1 recurrence (two 8-byte table reads per split at
// uniformly scattered subsets).  Each thread issues independent 8-byte loads
// from a 2^k-entry int64 table at indices drawn by a counter-based hash
// (SplitMix64, Steele et al. 2014), so nothing but the loads and the hash is
// timed; the loaded values are summed into one word so the loads are kept.
//
// mpt_alu_addmin_peak: the rate of the instruction the blocked recurrence
// spends its time in -- one 32-bit add fused with an unsigned min,
// acc = min(acc, x + y), one per split -- when nothing else competes for the
// integer ALU pipe.  Every SM runs 16 warps (4 per sub-partition); each
// thread keeps 32 running minima and updates each of them once per x value,
// acc[s] = min(acc[s], x[a] + y[s ^ a]) over all 32 x 32 (a, s): 1024
// independent add-min chains of distance 32 per step, every sum a different
// pair of registers.  Between steps the y values move by one through an
// integer multiply-add by a run-time one (the FMA pipe), so no sum repeats
// across steps and nothing in the loop can be hoisted.
#include <cstdint>

#include "../../include/mpt.h"
#include "mpt_internal.cuh"

namespace mpt {
namespace {

constexpr int kProbeThreads = 256;
constexpr int kProbeUnroll = 8;

__device__ __forceinline__ uint64_t splitmix64(uint64_t x) {
  x += 0x9E3779B97F4A7C15ull;
  x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
  x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
  return x ^ (x >> 31);
}

__global__ void __launch_bounds__(kProbeThreads)
k_gather_probe(const int64_t* __restrict__ table, uint64_t mask, int64_t per_thread, unsigned long long* __restrict__ sink) {
  const uint64_t tid = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  uint64_t ctr = tid * 0x100000001B3ull;
  int64_t acc = 0;
  for (int64_t i = 0; i < per_thread; i += kProbeUnroll) {
    int64_t v[kProbeUnroll];
#pragma unroll
    for (int u = 0; u < kProbeUnroll; ++u) v[u] = __ldcg(table + (splitmix64(ctr + (uint64_t)u) & mask));
#pragma unroll
    for (int u = 0; u < kProbeUnroll; ++u) acc += v[u];
    ctr += kProbeUnroll;
  }
  // entries are below 1024, so the sum never reaches 2^63 - 1: the test only keeps the loads alive
  if (acc == 0x7FFFFFFFFFFFFFFFll) atomicAdd(sink, 1ull);
}

__global__ void k_fill_probe(int64_t* __restrict__ table, uint64_t n) {
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (uint64_t)gridDim.x * blockDim.x)
    table[i] = (int64_t)(i & 1023);
}

constexpr int kAluThreads = 512;  // 16 warps per SM, 4 per sub-partition
constexpr int kAluRow = 32;       // running minima per thread
constexpr int kAluPerStep = kAluRow * kAluRow;

__global__ void __launch_bounds__(kAluThreads, 1)
k_addmin_probe(uint32_t seed, uint32_t one, int64_t steps, unsigned long long* __restrict__ sink) {
  const uint64_t tid = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  uint32_t x[kAluRow], y[kAluRow], acc[kAluRow];
#pragma unroll
  for (int j = 0; j < kAluRow; ++j) {
    const uint64_t h = splitmix64(((uint64_t)seed << 40) ^ (tid * kAluRow + (uint64_t)j));
    x[j] = (uint32_t)h & 0x1FFFFFFFu;
    y[j] = (uint32_t)(h >> 32) & 0x1FFFFFFFu;
    acc[j] = 0xFFFFFFFFu;
  }
  for (int64_t it = 0; it < steps; ++it) {
#pragma unroll
    for (int a = 0; a < kAluRow; ++a) {
#pragma unroll
      for (int s = 0; s < kAluRow; ++s) acc[s] = min(acc[s], x[a] + y[s ^ a]);
    }
#pragma unroll
    for (int j = 0; j < kAluRow; ++j) y[j] = y[j] * one + one;
  }
  uint32_t r = 0;
#pragma unroll
  for (int j = 0; j < kAluRow; ++j) r ^= acc[j];
  // never true: x < 2^29 and y < 2^29 + steps (steps < 2^28), so every minimum
  // is below 2^31 once the first sum is taken; it only keeps the minima alive
  if (r == 0xFFFFFFFFu) atomicAdd(sink, 1ull);
}

}  // namespace
}  // namespace mpt

extern "C" mpt_status mpt_alu_addmin_peak(int64_t ops, void* stream_ptr, double* ops_per_s) {
  using namespace mpt;
  if (!ops_per_s || ops < 1) return MPT_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream_ptr);
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return MPT_ERR_CUDA;
  const int64_t threads = (int64_t)sms * kAluThreads;
  const int64_t steps = (ops + threads * kAluPerStep - 1) / (threads * kAluPerStep);
  if (steps >= ((int64_t)1 << 28)) return MPT_ERR_INVALID_ARG;
  unsigned long long* sink = nullptr;
  if (device_alloc(reinterpret_cast<void**>(&sink), sizeof(unsigned long long)) != cudaSuccess)
    return MPT_ERR_OUT_OF_MEMORY;
  cudaEvent_t a = nullptr, b = nullptr;
  mpt_status status = MPT_OK;
  float ms = 0.f;
  if (cudaEventCreate(&a) != cudaSuccess || cudaEventCreate(&b) != cudaSuccess) {
    status = MPT_ERR_CUDA;
  } else {
    cudaMemsetAsync(sink, 0, sizeof(unsigned long long), st);
    const int64_t warm = steps < 64 ? steps : 64;
    k_addmin_probe<<<(unsigned)sms, kAluThreads, 0, st>>>(1u, 1u, warm, sink);
    cudaEventRecord(a, st);
    k_addmin_probe<<<(unsigned)sms, kAluThreads, 0, st>>>(2u, 1u, steps, sink);
    cudaEventRecord(b, st);
    if (cudaGetLastError() != cudaSuccess || cudaEventSynchronize(b) != cudaSuccess ||
        cudaEventElapsedTime(&ms, a, b) != cudaSuccess || ms <= 0.f)
      status = MPT_ERR_CUDA;
  }
  if (a) cudaEventDestroy(a);
  if (b) cudaEventDestroy(b);
  cudaFree(sink);
  if (status != MPT_OK) return status;
  *ops_per_s = (double)threads * (double)steps * (double)kAluPerStep / ((double)ms * 1e-3);
  return MPT_OK;
}

extern "C" mpt_status mpt_gather_bandwidth(int32_t log2_entries, int64_t loads, void* stream_ptr, double* gbps) {
  using namespace mpt;
  if (!gbps || log2_entries < 10 || log2_entries > 32 || loads < 1) return MPT_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream_ptr);
  const uint64_t n = (uint64_t)1 << log2_entries;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return MPT_ERR_CUDA;
  const int64_t blocks = (int64_t)sms * 16;
  const int64_t threads = blocks * kProbeThreads;
  int64_t per_thread = (loads + threads - 1) / threads;
  per_thread = (per_thread + kProbeUnroll - 1) / kProbeUnroll * kProbeUnroll;
  char* mem = nullptr;
  if (device_alloc(reinterpret_cast<void**>(&mem), n * 8 + 256) != cudaSuccess) return MPT_ERR_OUT_OF_MEMORY;
  int64_t* table = reinterpret_cast<int64_t*>(mem);
  unsigned long long* sink = reinterpret_cast<unsigned long long*>(mem + n * 8);
  cudaEvent_t a = nullptr, b = nullptr;
  mpt_status status = MPT_OK;
  float ms = 0.f;
  if (cudaEventCreate(&a) != cudaSuccess || cudaEventCreate(&b) != cudaSuccess) {
    status = MPT_ERR_CUDA;
  } else {
    k_fill_probe<<<(unsigned)blocks, kProbeThreads, 0, st>>>(table, n);
    cudaMemsetAsync(sink, 0, 8, st);
    k_gather_probe<<<(unsigned)blocks, kProbeThreads, 0, st>>>(table, n - 1, per_thread, sink);  // warm-up
    cudaEventRecord(a, st);
    k_gather_probe<<<(unsigned)blocks, kProbeThreads, 0, st>>>(table, n - 1, per_thread, sink);
    cudaEventRecord(b, st);
    if (cudaEventSynchronize(b) != cudaSuccess || cudaEventElapsedTime(&ms, a, b) != cudaSuccess || ms <= 0.f)
      status = MPT_ERR_CUDA;
  }
  if (a) cudaEventDestroy(a);
  if (b) cudaEventDestroy(b);
  cudaFree(mem);
  if (status != MPT_OK) return status;
  *gbps = (double)threads * (double)per_thread * 8.0 / ((double)ms * 1e-3) / 1e9;
  return MPT_OK;
}
