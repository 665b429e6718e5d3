// K3 (general form): the Sec. 3.1 recurrence with int64 values,
//     F({i}) = w(R_i),   F(S) = min over S = A (+) B of F(A) + F(B) - w(I(S)),
// one launch per popcount layer k = 2..m; every subset of a layer is
// independent.  A split is named by its part A holding the lowest request of
// S; A runs over those parts in increasing order and ties keep the smallest.
//
// This form reads F(A) and F(S \ A) straight from the 2^m table in HBM/L2 for
// every split (16 bytes per split), so it is bound by random gathers.  It is
// exact for any weights below the int64 limit and is used when the blocked
// kernels' packed keys could overflow (shared weight >= 2^51), or on
// request.  T is the table type: int64 (separate w(I) and F tables), or int32
// for the lean table, where wI and F are the same array -- the thread that
// finishes S reads w(I(S)) and writes F(S) over it, and F is read only at
// finished subsets of lower layers.
#include <climits>

#include "mpt_internal.cuh"

namespace mpt {
namespace {

constexpr int kThreads = 256;
constexpr int kThreadMaxLayer = 9;  // layers up to 9 requests: one subset per thread

template <typename T>
__global__ void k_dp_init(int m, const T* wI, T* F, uint32_t* __restrict__ split) {
  const int i = threadIdx.x;
  if (i == 0) {
    F[0] = 0;
    split[0] = 0;
  }
  if (i < m) {
    const uint32_t S = 1u << i;
    F[S] = wI[S];
    split[S] = 0;
  }
}

template <typename T>
__device__ __forceinline__ void scan_splits(uint32_t S, uint32_t low, uint32_t fixed, uint32_t free_bits,
                                            uint32_t rest, const T* F, int64_t& best, uint32_t& arg) {
  uint32_t sub = 0;
  do {
    const uint32_t part = fixed | sub;
    if (part != rest) {
      const uint32_t A = low | part;
      const int64_t c = (int64_t)F[A] + (int64_t)F[S ^ A];
      if (c < best) {
        best = c;
        arg = A;
      }
    }
    sub = (sub - free_bits) & free_bits;
  } while (sub != 0);
}

template <typename T>
__global__ void __launch_bounds__(kThreads)
k_dp_layer_thread(int m, int k, unsigned long long count, const T* wI, T* F, uint32_t* __restrict__ split,
                  int32_t* __restrict__ flags) {
  const unsigned long long idx = (unsigned long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= count) return;
  const uint32_t S = colex_unrank(idx, k, m);
  if (MPT_BAD(flags, (unsigned long long)S < (1ull << m) && __popc(S) == k)) return;
  const uint32_t low = S & (~S + 1u);
  const uint32_t rest = S ^ low;
  int64_t best = LLONG_MAX;
  uint32_t arg = 0;
  scan_splits(S, low, 0u, rest, rest, F, best, arg);
  if (MPT_BAD(flags, valid_split(S, arg))) return;
  F[S] = (T)(best - (int64_t)wI[S]);
  split[S] = arg;
}

// One warp per subset: lane r takes the parts whose top five bits (within S
// minus its lowest request) spell r; the lanes' results are merged
// lexicographically on (value, A).
template <typename T>
__global__ void __launch_bounds__(kThreads)
k_dp_layer_warp(int m, int k, unsigned long long count, const T* wI, T* F, uint32_t* __restrict__ split,
                int32_t* __restrict__ flags) {
  const int lane = threadIdx.x & 31;
  const unsigned long long warps = (unsigned long long)gridDim.x * (blockDim.x >> 5);
  for (unsigned long long w = (unsigned long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); w < count;
       w += warps) {
    const uint32_t S = colex_unrank(w, k, m);
    if (MPT_BAD(flags, (unsigned long long)S < (1ull << m) && __popc(S) == k)) continue;  // the same in every lane
    const uint32_t low = S & (~S + 1u);
    const uint32_t rest = S ^ low;
    uint32_t hi = 0, r = rest;
    for (int t = 0; t < 5; ++t) {
      const uint32_t top = 1u << (31 - __clz(r));
      hi |= top;
      r ^= top;
    }
    const uint32_t fixed = deposit_bits((uint32_t)lane, hi);
    int64_t best = LLONG_MAX;
    uint32_t arg = 0xFFFFFFFFu;
    scan_splits(S, low, fixed, rest ^ hi, rest, F, best, arg);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const int64_t ob = __shfl_xor_sync(0xFFFFFFFFu, best, off);
      const uint32_t oa = __shfl_xor_sync(0xFFFFFFFFu, arg, off);
      if (ob < best || (ob == best && oa < arg)) {
        best = ob;
        arg = oa;
      }
    }
    if (lane == 0 && !MPT_BAD(flags, valid_split(S, arg))) {
      F[S] = (T)(best - (int64_t)wI[S]);
      split[S] = arg;
    }
  }
}

template <typename T>
cudaError_t dp_general(const Shape& s, const T* wI, T* F, uint32_t* split, int32_t* flags, cudaStream_t stream,
                       int* launches, int step_begin, int step_end) {
  if (step_end < 0 || step_end > s.m) step_end = s.m;
  const int64_t sms = sm_count();
  cudaError_t err = cudaSuccess;
  if (step_begin <= 0 && step_end > 0) {
    k_dp_init<<<1, 32, 0, stream>>>(s.m, wI, F, split);
    ++*launches;
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
  }
  // step j >= 1 is the layer of (j + 1)-request subsets
  const int k_begin = step_begin < 1 ? 2 : step_begin + 1;
  for (int k = k_begin; k <= step_end; ++k) {
    const unsigned long long count = h_binom.v[s.m][k];
    if (k <= kThreadMaxLayer) {
      const unsigned long long blocks = (count + kThreads - 1) / kThreads;
      k_dp_layer_thread<<<(unsigned)blocks, kThreads, 0, stream>>>(s.m, k, count, wI, F, split, flags);
    } else {
      unsigned long long blocks = (count + (kThreads / 32) - 1) / (kThreads / 32);
      if (blocks > (unsigned long long)sms * 16) blocks = (unsigned long long)sms * 16;
      k_dp_layer_warp<<<(unsigned)blocks, kThreads, 0, stream>>>(s.m, k, count, wI, F, split, flags);
    }
    ++*launches;
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
  }
  return cudaSuccess;
}

}  // namespace

int dp_steps(const Shape& s) { return s.blocked ? s.L + 1 : s.m; }

cudaError_t launch_dp_general(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches,
                              int step_begin, int step_end) {
  if (s.lean)
    return dp_general<int32_t>(s, ws.fw, ws.fw, ws.split, ws.counters + 1, stream, launches, step_begin, step_end);
  return dp_general<int64_t>(s, ws.wI, ws.F, ws.split, ws.counters + 1, stream, launches, step_begin, step_end);
}

}  // namespace mpt
