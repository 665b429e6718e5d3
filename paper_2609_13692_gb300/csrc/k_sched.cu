// Serving order and finite radix cache (Sec. 8, Thm 7), and eq. (1) for many
// strings.
//
// Strings are laid-out requests (chunk ids).  Everything here starts from
// their lexicographic order (a string before its extensions), built by a
// stable least-significant-digit radix sort over string positions:
//   * Thm 7's serving order is that order (the DFS order of the trie), or,
//     with a bounded reorder window, that order inside each window;
//   * the trie of eq. (1): in lexicographic order, string x shares exactly
//     lcp[x] = lcp(string x-1, string x) nodes with all earlier strings, so
//     the trie weight is sum_x w(suffix of x after lcp[x]), and the node of
//     (x, depth s) is the one created by the last y <= x with lcp[y] <= s;
//   * the radix cache with LRU leaf eviction (Sec. 8).  Serving a request
//     touches every node on its root path; a node's last touch is never older
//     than its descendants', so the least recently used leaf is the least
//     recently used node, deepest first among a request's own path.  Evicting
//     in that order keeps the cache equal to the longest prefix of the
//     recency order (last touch descending, depth ascending) whose weight fits
//     the capacity C.  A node on request t's path is therefore a hit iff the
//     weight of the recency order up to and including it, d, is <= C -- one
//     number per access serves every capacity at once.  For the node v at
//     depth q of request t, last touched by request j < t,
//         d = sum over r in (j, t) of w(nodes of r's path not touched again before t)
//           + w(ancestors-or-self of v whose last touch before t is j).
#include <climits>
#include <cstring>
#include <vector>

#include "../../include/mpt.h"
#include "mpt_internal.cuh"

namespace mpt {
namespace {

// ---------------------------------------------------------------------------
// Stable LSD radix sort of (uint32 key, uint32 value) pairs, 8 bits a pass.
// A tile of 2048 keys per block; pass = digit histogram per tile, exclusive
// scan of the digit-major [256][tiles] counts, stable scatter.
// ---------------------------------------------------------------------------
constexpr int kRsThreads = 256;
constexpr int kRsRounds = 8;
constexpr int kRsTile = kRsThreads * kRsRounds;
constexpr int kRsBins = 256;
constexpr int kRsWarps = kRsThreads / 32;

__global__ void __launch_bounds__(kRsThreads)
k_rs_hist(const uint32_t* __restrict__ keys, int64_t n, int shift, uint32_t* __restrict__ hist, int tiles) {
  __shared__ uint32_t h[kRsBins];
  h[threadIdx.x] = 0;
  __syncthreads();
  const int64_t start = (int64_t)blockIdx.x * kRsTile;
  for (int i = threadIdx.x; i < kRsTile; i += kRsThreads) {
    const int64_t idx = start + i;
    if (idx < n) atomicAdd(&h[(keys[idx] >> shift) & 0xFFu], 1u);
  }
  __syncthreads();
  hist[(int64_t)threadIdx.x * tiles + blockIdx.x] = h[threadIdx.x];
}

__global__ void __launch_bounds__(kRsThreads)
k_rs_scatter(const uint32_t* __restrict__ kin, const uint32_t* __restrict__ vin, uint32_t* __restrict__ kout,
             uint32_t* __restrict__ vout, int64_t n, int shift, const uint32_t* __restrict__ offs, int tiles) {
  __shared__ uint32_t base[kRsBins];
  __shared__ uint32_t tot[kRsBins];
  __shared__ uint32_t wcnt[kRsWarps][kRsBins];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  base[tid] = offs[(int64_t)tid * tiles + blockIdx.x];
  const int64_t start = (int64_t)blockIdx.x * kRsTile;
  const uint32_t lt = (1u << lane) - 1u;
  for (int round = 0; round < kRsRounds; ++round) {
#pragma unroll
    for (int w = 0; w < kRsWarps; ++w) wcnt[w][tid] = 0;
    __syncthreads();
    const int64_t idx = start + (int64_t)round * kRsThreads + tid;
    const bool valid = idx < n;
    uint32_t key = 0, val = 0, digit = 0xFFFFu;  // 0xFFFF: no key (never a digit)
    if (valid) {
      key = kin[idx];
      val = vin[idx];
      digit = (key >> shift) & 0xFFu;
    }
    const uint32_t peers = __match_any_sync(0xFFFFFFFFu, digit);
    const uint32_t rank = __popc(peers & lt);
    if (valid && rank == 0) wcnt[warp][digit] = __popc(peers);
    __syncthreads();
    {
      uint32_t run = 0;
#pragma unroll
      for (int w = 0; w < kRsWarps; ++w) {
        const uint32_t c = wcnt[w][tid];
        wcnt[w][tid] = run;
        run += c;
      }
      tot[tid] = run;
    }
    __syncthreads();
    if (valid) {
      const uint32_t pos = base[digit] + wcnt[warp][digit] + rank;
      kout[pos] = key;
      vout[pos] = val;
    }
    __syncthreads();
    base[tid] += tot[tid];
  }
}

// Exclusive prefix sum of uint32 values in place (n <= 2048 * 16384).
constexpr int kScanThreads = 256;
constexpr int kScanItems = 8;
constexpr int kScanTile = kScanThreads * kScanItems;
constexpr int kScanSumThreads = 1024;
constexpr int kScanSumItems = 16;

template <int kThreads>
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* total) {
  __shared__ uint32_t warp_sums[kThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    uint32_t s = lane < kThreads / 32 ? warp_sums[lane] : 0u;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, s, off);
      if (lane >= off) s += y;
    }
    if (lane < kThreads / 32) warp_sums[lane] = s;
  }
  __syncthreads();
  const uint32_t before = (warp > 0 ? warp_sums[warp - 1] : 0u) + x - v;
  *total = warp_sums[kThreads / 32 - 1];
  __syncthreads();
  return before;
}

__global__ void __launch_bounds__(kScanThreads) k_scan_tiles(uint32_t* __restrict__ a, int64_t n, uint32_t* __restrict__ sums) {
  const int64_t first = (int64_t)blockIdx.x * kScanTile + (int64_t)threadIdx.x * kScanItems;
  uint32_t v[kScanItems];
  uint32_t local = 0;
#pragma unroll
  for (int i = 0; i < kScanItems; ++i) {
    v[i] = first + i < n ? a[first + i] : 0u;
    local += v[i];
  }
  uint32_t total;
  uint32_t run = block_exclusive_scan<kScanThreads>(local, &total);
#pragma unroll
  for (int i = 0; i < kScanItems; ++i) {
    if (first + i < n) a[first + i] = run;
    run += v[i];
  }
  if (threadIdx.x == 0) sums[blockIdx.x] = total;
}

__global__ void __launch_bounds__(kScanSumThreads) k_scan_sums(uint32_t* __restrict__ sums, int count) {
  const int first = threadIdx.x * kScanSumItems;
  uint32_t v[kScanSumItems];
  uint32_t local = 0;
#pragma unroll
  for (int i = 0; i < kScanSumItems; ++i) {
    v[i] = first + i < count ? sums[first + i] : 0u;
    local += v[i];
  }
  uint32_t total;
  uint32_t run = block_exclusive_scan<kScanSumThreads>(local, &total);
#pragma unroll
  for (int i = 0; i < kScanSumItems; ++i) {
    if (first + i < count) sums[first + i] = run;
    run += v[i];
  }
}

__global__ void __launch_bounds__(kScanThreads) k_scan_add(uint32_t* __restrict__ a, int64_t n, const uint32_t* __restrict__ sums) {
  const int64_t first = (int64_t)blockIdx.x * kScanTile;
  const uint32_t add = sums[blockIdx.x];
  for (int i = threadIdx.x; i < kScanTile; i += kScanThreads) {
    const int64_t idx = first + i;
    if (idx < n) a[idx] += add;
  }
}

constexpr int64_t kScanMax = (int64_t)kScanTile * kScanSumThreads * kScanSumItems;

int64_t scan_tiles(int64_t n) { return (n + kScanTile - 1) / kScanTile; }

cudaError_t exclusive_scan(uint32_t* a, int64_t n, uint32_t* sums, cudaStream_t st, int* launches) {
  if (n <= 0) return cudaSuccess;
  if (n > kScanMax) return cudaErrorInvalidValue;
  const int tiles = (int)scan_tiles(n);
  k_scan_tiles<<<tiles, kScanThreads, 0, st>>>(a, n, sums);
  k_scan_sums<<<1, kScanSumThreads, 0, st>>>(sums, tiles);
  k_scan_add<<<tiles, kScanThreads, 0, st>>>(a, n, sums);
  *launches += 3;
  return cudaGetLastError();
}

int64_t rs_tiles(int64_t n) { return (n + kRsTile - 1) / kRsTile; }

// Scratch of a radix sort of n pairs: second key/value buffers, the digit
// counts and the scan's tile sums.
struct SortScratch {
  uint32_t* k2;
  uint32_t* v2;
  uint32_t* hist;
  uint32_t* sums;
};

// Sort (*keys, *vals) by key bits [0, bits); the sorted arrays end up in
// *keys / *vals (the pointers may be swapped with the scratch buffers).
cudaError_t radix_sort(uint32_t** keys, uint32_t** vals, SortScratch& s, int64_t n, int bits, cudaStream_t st,
                       int* launches) {
  if (n <= 1 || bits <= 0) return cudaSuccess;
  const int tiles = (int)rs_tiles(n);
  for (int shift = 0; shift < bits; shift += 8) {
    k_rs_hist<<<tiles, kRsThreads, 0, st>>>(*keys, n, shift, s.hist, tiles);
    ++*launches;
    cudaError_t e = exclusive_scan(s.hist, (int64_t)kRsBins * tiles, s.sums, st, launches);
    if (e != cudaSuccess) return e;
    k_rs_scatter<<<tiles, kRsThreads, 0, st>>>(*keys, *vals, s.k2, s.v2, n, shift, s.hist, tiles);
    ++*launches;
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    uint32_t* t = *keys;
    *keys = s.k2;
    s.k2 = t;
    t = *vals;
    *vals = s.v2;
    s.v2 = t;
  }
  return cudaSuccess;
}

int bits_for(uint64_t max_value) {
  int b = 0;
  while (b < 64 && (max_value >> b) != 0) ++b;
  return b;
}

// ---------------------------------------------------------------------------
// Lexicographic order of the strings.
// ---------------------------------------------------------------------------
constexpr int kThreads = 256;

// blocks of kThreads for n items, at most per_sm per SM (grid-stride loops)
unsigned grid_for(int64_t n, int64_t per_sm = 32) {
  int64_t b = (n + kThreads - 1) / kThreads;
  const int64_t cap = sm_count() * per_sm;
  if (b > cap) b = cap;
  return (unsigned)(b < 1 ? 1 : b);
}

__global__ void k_iota(uint32_t* __restrict__ a, int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    a[i] = (uint32_t)i;
}

// key of the string at sorted position i for position s: chunk + 1, or 0 past its end
__global__ void k_lex_keys(const uint32_t* __restrict__ ord, int64_t m, const int64_t* __restrict__ off,
                           const int32_t* __restrict__ chunk, int s, uint32_t* __restrict__ keys) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < m; i += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t r = ord[i];
    const int64_t b = off[r], len = off[r + 1] - b;
    keys[i] = s < len ? (uint32_t)chunk[b + s] + 1u : 0u;
  }
}

__global__ void k_inverse(const uint32_t* __restrict__ ord, int64_t m, int32_t* __restrict__ pos) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < m; i += (int64_t)gridDim.x * blockDim.x)
    pos[ord[i]] = (int32_t)i;
}

// lcp[x] = common prefix length of the strings at sorted positions x - 1 and x
// (lcp[0] = 0); trie weight = sum_x w(suffix of string x after lcp[x]).
__global__ void __launch_bounds__(kThreads)
k_lcp_cost(const uint32_t* __restrict__ ord, int64_t m, const int64_t* __restrict__ off,
           const int32_t* __restrict__ chunk, const int64_t* __restrict__ w, int32_t* __restrict__ lcp,
           unsigned long long* __restrict__ cost) {
  unsigned long long local = 0;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < m; x += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t r = ord[x];
    const int64_t b = off[r], len = off[r + 1] - b;
    int64_t l = 0;
    if (x > 0) {
      const uint32_t p = ord[x - 1];
      const int64_t pb = off[p], plen = off[p + 1] - pb;
      const int64_t lim = len < plen ? len : plen;
      while (l < lim && chunk[b + l] == chunk[pb + l]) ++l;
    }
    lcp[x] = (int32_t)l;
    for (int64_t s = l; s < len; ++s) local += (unsigned long long)w[chunk[b + s]];
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) local += __shfl_xor_sync(0xFFFFFFFFu, local, o);
  if ((threadIdx.x & 31) == 0 && local) atomicAdd(cost, local);
}

// ---------------------------------------------------------------------------
// Trie nodes and the per-access recency distance.
// ---------------------------------------------------------------------------
// st[k][i] = min lcp[i - 2^k + 1 .. i]  (k = 1 .. K-1; level 0 is lcp itself)
__global__ void k_sparse_level(int32_t* __restrict__ st, int64_t m, int k) {
  const int64_t half = (int64_t)1 << (k - 1);
  const int32_t* prev = st + (int64_t)(k - 1) * m;
  int32_t* cur = st + (int64_t)k * m;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < m; i += (int64_t)gridDim.x * blockDim.x) {
    const int32_t a = prev[i];
    cur[i] = i >= half ? min(a, prev[i - half]) : a;
  }
}

// the last sorted position y <= x with lcp[y] <= s (exists: lcp[0] = 0)
__device__ __forceinline__ int64_t node_owner(const int32_t* __restrict__ st, int64_t m, int K, int64_t x, int s) {
  if (st[x] <= s) return x;
  int64_t p = x;  // every lcp in [p, x] is > s
  for (int k = K - 1; k >= 0; --k) {
    const int64_t len = (int64_t)1 << k;
    if (p - len >= 0 && st[(int64_t)k * m + (p - 1)] > s) p -= len;
  }
  return p - 1;
}

// new[x] = nodes first created by the string at sorted position x
__global__ void k_new_nodes(const uint32_t* __restrict__ ord, int64_t m, const int64_t* __restrict__ off,
                            const int32_t* __restrict__ lcp, uint32_t* __restrict__ fresh) {
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < m; x += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t r = ord[x];
    fresh[x] = (uint32_t)(off[r + 1] - off[r] - lcp[x]);
  }
}

// Per access (served position t, depth s), laid out at aoff[t] + s: its trie
// node, its chunk weight, its request's served position.
__global__ void __launch_bounds__(kThreads)
k_accesses(const int32_t* __restrict__ order, int64_t m, const int64_t* __restrict__ off,
           const int32_t* __restrict__ chunk, const int64_t* __restrict__ w, const int32_t* __restrict__ lexpos,
           const int32_t* __restrict__ st, int K, const uint32_t* __restrict__ node_base,
           const int64_t* __restrict__ aoff, uint32_t* __restrict__ node, uint32_t* __restrict__ acc_id,
           int64_t* __restrict__ aw, int64_t* __restrict__ asuf, int32_t* __restrict__ aowner) {
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < m; t += (int64_t)gridDim.x * blockDim.x) {
    const int32_t r = order[t];
    const int64_t b = off[r], len = off[r + 1] - b;
    const int64_t x = lexpos[r];
    const int64_t a0 = aoff[t];
    for (int64_t s = 0; s < len; ++s) {
      const int64_t y = node_owner(st, m, K, x, (int)s);
      node[a0 + s] = node_base[y] + (uint32_t)(s - st[y]);
      acc_id[a0 + s] = (uint32_t)(a0 + s);
      aw[a0 + s] = w[chunk[b + s]];
      aowner[a0 + s] = (int32_t)t;
    }
    int64_t suf = 0;
    for (int64_t s = len - 1; s >= 0; --s) {
      suf += aw[a0 + s];
      asuf[a0 + s] = suf;
    }
  }
}

// After a stable sort of accesses by node (input in served order), neighbours
// with the same node are consecutive touches of it.
__global__ void k_prev_next(const uint32_t* __restrict__ skey, const uint32_t* __restrict__ sacc, int64_t N,
                            const int32_t* __restrict__ aowner, int32_t* __restrict__ prev_t,
                            int32_t* __restrict__ next_t) {
  for (int64_t z = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; z < N; z += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t a = sacc[z], k = skey[z];
    prev_t[a] = (z > 0 && skey[z - 1] == k) ? aowner[sacc[z - 1]] : -1;
    next_t[a] = (z + 1 < N && skey[z + 1] == k) ? aowner[sacc[z + 1]] : INT_MAX;
  }
}

// the largest capacity below the trie weight (every distance is at most the
// trie weight, so larger capacities see only compulsory misses)
__global__ void k_scan_limit(const int64_t* __restrict__ caps, int n_caps, const unsigned long long* __restrict__ trie,
                             int64_t* __restrict__ limit) {
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    int64_t best = -1;
    const int64_t tw = (int64_t)*trie;
    for (int i = 0; i < n_caps; ++i)
      if (caps[i] < tw && caps[i] > best) best = caps[i];
    *limit = best;
  }
}

// weight of the nodes of served request r's path not touched again before t
__device__ __forceinline__ int64_t untouched_suffix(const int64_t* __restrict__ aoff, const int32_t* __restrict__ next_t,
                                                    const int64_t* __restrict__ asuf, int64_t r, int64_t t) {
  const int64_t b = aoff[r];
  int64_t lo = 0, hi = aoff[r + 1] - b;  // next_t is nondecreasing along a path
  const int64_t len = hi;
  while (lo < hi) {
    const int64_t mid = (lo + hi) >> 1;
    if ((int64_t)next_t[b + mid] >= t)
      hi = mid;
    else
      lo = mid + 1;
  }
  return lo < len ? asuf[b + lo] : 0;
}

constexpr int kDistThreads = 256;

// One warp per served request t: the recency distance of each access on its
// path.  dist = INT64_MAX for a first touch (a miss at every capacity),
// limit + 1 when it exceeds the largest capacity of interest.
__global__ void __launch_bounds__(kDistThreads)
k_distance(int64_t m, const int64_t* __restrict__ aoff, const int32_t* __restrict__ prev_t,
           const int32_t* __restrict__ next_t, const int64_t* __restrict__ aw, const int64_t* __restrict__ asuf,
           const int64_t* __restrict__ limit_p, int64_t* __restrict__ dist) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kDistThreads / 32);
  const int64_t limit = *limit_p;
  for (int64_t t = (int64_t)blockIdx.x * (kDistThreads / 32) + (threadIdx.x >> 5); t < m; t += warps) {
    const int64_t b = aoff[t], len = aoff[t + 1] - b;
    int64_t scanned = t;  // requests [scanned, t) are summed
    int64_t sum = 0;
    bool over = limit < 0;
    int64_t run_j = -2, run_w = 0;
    for (int64_t q = 0; q < len; ++q) {
      const int64_t j = prev_t[b + q];
      int64_t d;
      if (j < 0) {
        d = LLONG_MAX;
      } else {
        const int64_t wq = aw[b + q];
        if (j == run_j) {
          run_w += wq;
        } else {
          run_j = j;
          run_w = wq;
        }
        while (!over && scanned > j + 1) {
          const int64_t lo = scanned - 32 > j + 1 ? scanned - 32 : j + 1;
          const int64_t r = scanned - 1 - lane;
          int64_t c = r >= lo ? untouched_suffix(aoff, next_t, asuf, r, t) : 0;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xFFFFFFFFu, c, o);
          sum += c;
          scanned = lo;
          if (sum > limit) over = true;
        }
        d = over ? limit + 1 : sum + run_w;
        if (d > limit) d = limit + 1;
      }
      if (lane == 0) dist[b + q] = d;
    }
  }
}

constexpr int kMaxCaps = 1024;

__global__ void __launch_bounds__(kThreads)
k_cache_costs(const int64_t* __restrict__ dist, const int64_t* __restrict__ aw, int64_t N,
              const int64_t* __restrict__ caps, int n_caps, unsigned long long* __restrict__ costs,
              unsigned long long* __restrict__ compulsory) {
  __shared__ unsigned long long acc[kMaxCaps];
  __shared__ int64_t cap_s[kMaxCaps];
  for (int i = threadIdx.x; i < n_caps; i += blockDim.x) {
    acc[i] = 0;
    cap_s[i] = caps[i];
  }
  __syncthreads();
  unsigned long long first = 0;
  for (int64_t a = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; a < N; a += (int64_t)gridDim.x * blockDim.x) {
    const int64_t d = dist[a];
    const unsigned long long wa = (unsigned long long)aw[a];
    if (d == LLONG_MAX) first += wa;
    for (int i = 0; i < n_caps; ++i)
      if (d > cap_s[i]) atomicAdd(&acc[i], wa);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) first += __shfl_xor_sync(0xFFFFFFFFu, first, o);
  if ((threadIdx.x & 31) == 0 && first) atomicAdd(compulsory, first);
  __syncthreads();
  for (int i = threadIdx.x; i < n_caps; i += blockDim.x)
    if (acc[i]) atomicAdd(&costs[i], acc[i]);
}

// order[z] = arrival[vals[z]]
__global__ void k_gather_order(const uint32_t* __restrict__ vals, const int32_t* __restrict__ arrival, int64_t m,
                               int32_t* __restrict__ order) {
  for (int64_t z = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; z < m; z += (int64_t)gridDim.x * blockDim.x)
    order[z] = arrival[vals[z]];
}

__global__ void k_window_keys(const uint32_t* __restrict__ vals, const int32_t* __restrict__ arrival,
                              const int32_t* __restrict__ lexpos, int64_t m, int64_t window, int pass,
                              uint32_t* __restrict__ keys) {
  for (int64_t z = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; z < m; z += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t a = vals[z];
    keys[z] = pass == 0 ? (uint32_t)lexpos[arrival[a]] : (uint32_t)((int64_t)a / window);
  }
}

// ---------------------------------------------------------------------------
// Host side.
// ---------------------------------------------------------------------------
constexpr int64_t kMaxStrings = (int64_t)1 << 22;
constexpr int64_t kMaxAccesses = (int64_t)1 << 27;
constexpr int64_t kMaxLength = 4096;

struct Arena {
  char* base = nullptr;
  size_t off = 0;
  template <typename T>
  T* take(int64_t count) {
    T* p = reinterpret_cast<T*>(base ? base + off : nullptr);
    off += ((size_t)(count > 0 ? count : 1) * sizeof(T) + 255) & ~(size_t)255;
    return p;
  }
};

struct Strings {
  int64_t m = 0, total = 0, maxlen = 0;
  std::vector<int32_t> chunk;
};

mpt_status check_strings(int64_t n_chunks, int64_t m, const int64_t* offsets, const int64_t* chunks, Strings* out) {
  if (!offsets || n_chunks < 1 || n_chunks >= INT32_MAX || m < 1) return MPT_ERR_INVALID_ARG;
  if (m > kMaxStrings) return MPT_ERR_TOO_LARGE;
  if (offsets[0] != 0) return MPT_ERR_INVALID_ARG;
  int64_t maxlen = 0;
  for (int64_t i = 0; i < m; ++i) {
    const int64_t len = offsets[i + 1] - offsets[i];
    if (len < 0) return MPT_ERR_INVALID_ARG;
    if (len > maxlen) maxlen = len;
  }
  const int64_t total = offsets[m];
  if (total > 0 && !chunks) return MPT_ERR_INVALID_ARG;
  if (total > kMaxAccesses || maxlen > kMaxLength) return MPT_ERR_TOO_LARGE;
  out->m = m;
  out->total = total;
  out->maxlen = maxlen;
  try {
    out->chunk.resize((size_t)(total > 0 ? total : 1));
  } catch (...) {
    return MPT_ERR_OUT_OF_MEMORY;
  }
  for (int64_t p = 0; p < total; ++p) {
    if (chunks[p] < 0 || chunks[p] >= n_chunks) return MPT_ERR_INVALID_ARG;
    out->chunk[(size_t)p] = (int32_t)chunks[p];
  }
  return MPT_OK;
}

mpt_status check_weights(const int64_t* weights, int64_t n_chunks) {
  if (!weights) return MPT_ERR_INVALID_ARG;
  for (int64_t x = 0; x < n_chunks; ++x)
    if (weights[x] <= 0) return MPT_ERR_INVALID_ARG;
  return MPT_OK;
}

mpt_status check_permutation(const int32_t* p, int64_t m) {
  std::vector<char> seen((size_t)m, 0);
  for (int64_t i = 0; i < m; ++i) {
    if (p[i] < 0 || p[i] >= m || seen[(size_t)p[i]]) return MPT_ERR_INVALID_ARG;
    seen[(size_t)p[i]] = 1;
  }
  return MPT_OK;
}

// Device copies of the strings and the buffers of their lexicographic sort.
struct LexBuffers {
  int64_t* off;
  int32_t* chunk;
  int64_t* w;
  uint32_t* keys;
  uint32_t* ord;
  SortScratch sort;
  int32_t* lexpos;
  int32_t* lcp;  // level 0 of the sparse table when the cache is simulated
  unsigned long long* trie;
};

void carve_lex(Arena& a, const Strings& s, int64_t n_chunks, int64_t sparse_levels, bool weights, LexBuffers* b) {
  const int64_t m = s.m;
  b->off = a.take<int64_t>(m + 1);
  b->chunk = a.take<int32_t>(s.total);
  b->w = weights ? a.take<int64_t>(n_chunks) : nullptr;
  b->keys = a.take<uint32_t>(m);
  b->ord = a.take<uint32_t>(m);
  b->sort.k2 = a.take<uint32_t>(m);
  b->sort.v2 = a.take<uint32_t>(m);
  b->sort.hist = a.take<uint32_t>((int64_t)kRsBins * rs_tiles(m));
  b->sort.sums = a.take<uint32_t>(scan_tiles((int64_t)kRsBins * rs_tiles(m)));
  b->lexpos = a.take<int32_t>(m);
  b->lcp = a.take<int32_t>(m * (sparse_levels > 0 ? sparse_levels : 1));
  b->trie = a.take<unsigned long long>(1);
}

// Sorts the strings (b->ord = string at each sorted position, b->lexpos its
// inverse); with weights, also lcp and the trie weight.
cudaError_t run_lex(const Strings& s, LexBuffers* b, int n_bits, bool with_cost, cudaStream_t st, int* launches) {
  const int64_t m = s.m;
  k_iota<<<grid_for(m), kThreads, 0, st>>>(b->ord, m);
  ++*launches;
  for (int64_t pos = s.maxlen - 1; pos >= 0; --pos) {
    k_lex_keys<<<grid_for(m), kThreads, 0, st>>>(b->ord, m, b->off, b->chunk, (int)pos, b->keys);
    ++*launches;
    cudaError_t e = radix_sort(&b->keys, &b->ord, b->sort, m, n_bits, st, launches);
    if (e != cudaSuccess) return e;
  }
  k_inverse<<<grid_for(m), kThreads, 0, st>>>(b->ord, m, b->lexpos);
  ++*launches;
  if (with_cost) {
    cudaError_t e = cudaMemsetAsync(b->trie, 0, sizeof(unsigned long long), st);
    if (e != cudaSuccess) return e;
    k_lcp_cost<<<grid_for(m), kThreads, 0, st>>>(b->ord, m, b->off, b->chunk, b->w, b->lcp, b->trie);
    ++*launches;
  }
  return cudaGetLastError();
}

cudaError_t upload_strings(const Strings& s, const int64_t* offsets, const int64_t* weights, int64_t n_chunks,
                           LexBuffers* b, cudaStream_t st) {
  cudaError_t e = cudaMemcpyAsync(b->off, offsets, (size_t)(s.m + 1) * 8, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess && s.total > 0)
    e = cudaMemcpyAsync(b->chunk, s.chunk.data(), (size_t)s.total * 4, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess && b->w) e = cudaMemcpyAsync(b->w, weights, (size_t)n_chunks * 8, cudaMemcpyHostToDevice, st);
  return e;
}

mpt_status cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return MPT_OK;
  return e == cudaErrorMemoryAllocation ? MPT_ERR_OUT_OF_MEMORY : MPT_ERR_CUDA;
}

int sparse_levels_for(int64_t m) {
  int K = 1;
  while (((int64_t)1 << K) <= m) ++K;
  return K;  // 2^K > m
}

}  // namespace

// Eq. (1) for any number of strings (used by mpt_trie_cost beyond 32 strings).
mpt_status trie_cost_lex(const int64_t* weights, int64_t n_chunks, int64_t m, const int64_t* offsets,
                         const int64_t* chunks, cudaStream_t st, int64_t* cost) {
  Strings s;
  mpt_status ms = check_strings(n_chunks, m, offsets, chunks, &s);
  if (ms != MPT_OK) return ms;
  if ((ms = check_weights(weights, n_chunks)) != MPT_OK) return ms;
  Arena a;
  LexBuffers b{};
  carve_lex(a, s, n_chunks, 1, true, &b);
  char* mem = nullptr;
  cudaError_t e = device_alloc(reinterpret_cast<void**>(&mem), a.off);
  if (e != cudaSuccess) return cuda_status(e);
  Arena a2{mem, 0};
  carve_lex(a2, s, n_chunks, 1, true, &b);
  int launches = 0;
  unsigned long long h = 0;
  e = upload_strings(s, offsets, weights, n_chunks, &b, st);
  if (e == cudaSuccess) e = run_lex(s, &b, bits_for((uint64_t)n_chunks), true, st, &launches);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&h, b.trie, 8, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(mem);
  if (e != cudaSuccess) return cuda_status(e);
  *cost = (int64_t)h;
  return MPT_OK;
}

}  // namespace mpt

extern "C" {

mpt_status mpt_serve_order(int64_t n_chunks, int32_t m, const int64_t* seq_offsets, const int64_t* seq_chunks,
                           const int32_t* arrival, int32_t window, void* stream, int32_t* order) {
  using namespace mpt;
  if (!order) return MPT_ERR_INVALID_ARG;
  Strings s;
  mpt_status ms = check_strings(n_chunks, m, seq_offsets, seq_chunks, &s);
  if (ms != MPT_OK) return ms;
  if (arrival && (ms = check_permutation(arrival, m)) != MPT_OK) return ms;
  if (window < 0) return MPT_ERR_INVALID_ARG;
  const bool windowed = window > 0 && window < m;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);

  Arena a;
  LexBuffers b{};
  carve_lex(a, s, n_chunks, 1, false, &b);
  int32_t* d_arrival = a.take<int32_t>(m);
  int32_t* d_order = a.take<int32_t>(m);
  char* mem = nullptr;
  cudaError_t e = device_alloc(reinterpret_cast<void**>(&mem), a.off);
  if (e != cudaSuccess) return cuda_status(e);
  Arena a2{mem, 0};
  carve_lex(a2, s, n_chunks, 1, false, &b);
  d_arrival = a2.take<int32_t>(m);
  d_order = a2.take<int32_t>(m);

  std::vector<int32_t> ident;
  const int32_t* arr = arrival;
  if (!arr) {
    ident.resize((size_t)m);
    for (int32_t i = 0; i < m; ++i) ident[(size_t)i] = i;
    arr = ident.data();
  }
  int launches = 0;
  e = upload_strings(s, seq_offsets, nullptr, n_chunks, &b, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(d_arrival, arr, (size_t)m * 4, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = run_lex(s, &b, bits_for((uint64_t)n_chunks), false, st, &launches);
  if (e == cudaSuccess) {
    if (!windowed) {
      e = cudaMemcpyAsync(d_order, b.ord, (size_t)m * 4, cudaMemcpyDeviceToDevice, st);
    } else {
      // sort arrival positions by (window index, lexicographic position)
      uint32_t* keys = b.keys;
      uint32_t* vals = b.ord;
      k_iota<<<grid_for(m), kThreads, 0, st>>>(vals, m);
      for (int pass = 0; pass < 2 && e == cudaSuccess; ++pass) {
        k_window_keys<<<grid_for(m), kThreads, 0, st>>>(vals, d_arrival, b.lexpos, m, window, pass, keys);
        const int nb = pass == 0 ? bits_for((uint64_t)m) : bits_for((uint64_t)((m - 1) / window));
        e = radix_sort(&keys, &vals, b.sort, m, nb, st, &launches);
      }
      if (e == cudaSuccess) k_gather_order<<<grid_for(m), kThreads, 0, st>>>(vals, d_arrival, m, d_order);
      if (e == cudaSuccess) e = cudaGetLastError();
    }
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(order, d_order, (size_t)m * 4, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(mem);
  return cuda_status(e);
}

mpt_status mpt_cache_costs(const int64_t* weights, int64_t n_chunks, int32_t m, const int64_t* seq_offsets,
                           const int64_t* seq_chunks, const int32_t* order, const int64_t* capacities,
                           int32_t n_caps, void* stream, int64_t* costs, int64_t* unbounded) {
  using namespace mpt;
  if (n_caps < 0 || n_caps > kMaxCaps || (n_caps > 0 && (!capacities || !costs))) return MPT_ERR_INVALID_ARG;
  for (int32_t i = 0; i < n_caps; ++i)
    if (capacities[i] < 0) return MPT_ERR_INVALID_ARG;
  Strings s;
  mpt_status ms = check_strings(n_chunks, m, seq_offsets, seq_chunks, &s);
  if (ms != MPT_OK) return ms;
  if ((ms = check_weights(weights, n_chunks)) != MPT_OK) return ms;
  if (order && (ms = check_permutation(order, m)) != MPT_OK) return ms;
  {
    // distances and costs are sums of distinct node weights: bounded by the
    // total string weight
    int64_t total_w = 0;
    for (int64_t p = 0; p < s.total; ++p) {
      const int64_t wx = weights[s.chunk[(size_t)p]];
      if (total_w > ((int64_t)1 << 62) - wx) return MPT_ERR_OVERFLOW;
      total_w += wx;
    }
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int64_t N = s.total;
  const int K = sparse_levels_for(m);

  std::vector<int32_t> h_order((size_t)m);
  std::vector<int64_t> h_aoff((size_t)m + 1);
  for (int32_t t = 0; t < m; ++t) h_order[(size_t)t] = order ? order[t] : t;
  h_aoff[0] = 0;
  for (int32_t t = 0; t < m; ++t) {
    const int32_t r = h_order[(size_t)t];
    h_aoff[(size_t)t + 1] = h_aoff[(size_t)t] + (seq_offsets[r + 1] - seq_offsets[r]);
  }

  auto carve = [&](Arena& a, LexBuffers* b, int32_t** d_order, int64_t** d_aoff, uint32_t** node_base,
                   uint32_t** node, uint32_t** acc_id, SortScratch* as, int64_t** aw, int64_t** asuf,
                   int32_t** aowner, int32_t** prev_t, int32_t** next_t, int64_t** dist, int64_t** d_caps,
                   int64_t** limit, unsigned long long** d_costs, unsigned long long** compulsory) {
    carve_lex(a, s, n_chunks, K, true, b);
    *d_order = a.take<int32_t>(m);
    *d_aoff = a.take<int64_t>(m + 1);
    *node_base = a.take<uint32_t>(m);
    *node = a.take<uint32_t>(N);
    *acc_id = a.take<uint32_t>(N);
    as->k2 = a.take<uint32_t>(N);
    as->v2 = a.take<uint32_t>(N);
    as->hist = a.take<uint32_t>((int64_t)kRsBins * rs_tiles(N));
    as->sums = a.take<uint32_t>(scan_tiles((int64_t)kRsBins * rs_tiles(N)) + scan_tiles(m));
    *aw = a.take<int64_t>(N);
    *asuf = a.take<int64_t>(N);
    *aowner = a.take<int32_t>(N);
    *prev_t = a.take<int32_t>(N);
    *next_t = a.take<int32_t>(N);
    *dist = a.take<int64_t>(N);
    *d_caps = a.take<int64_t>(n_caps);
    *limit = a.take<int64_t>(1);
    *d_costs = a.take<unsigned long long>(n_caps);
    *compulsory = a.take<unsigned long long>(1);
  };
  LexBuffers b{};
  int32_t* d_order;
  int64_t *d_aoff, *aw, *asuf, *dist, *d_caps, *limit;
  uint32_t *node_base, *node, *acc_id;
  SortScratch as{};
  int32_t *aowner, *prev_t, *next_t;
  unsigned long long *d_costs, *compulsory;
  Arena a;
  carve(a, &b, &d_order, &d_aoff, &node_base, &node, &acc_id, &as, &aw, &asuf, &aowner, &prev_t, &next_t, &dist,
        &d_caps, &limit, &d_costs, &compulsory);
  char* mem = nullptr;
  cudaError_t e = device_alloc(reinterpret_cast<void**>(&mem), a.off);
  if (e != cudaSuccess) return cuda_status(e);
  Arena a2{mem, 0};
  carve(a2, &b, &d_order, &d_aoff, &node_base, &node, &acc_id, &as, &aw, &asuf, &aowner, &prev_t, &next_t, &dist,
        &d_caps, &limit, &d_costs, &compulsory);

  int launches = 0;
  unsigned long long h_trie = 0, h_first = 0;
  std::vector<unsigned long long> h_costs((size_t)(n_caps > 0 ? n_caps : 1));
  e = upload_strings(s, seq_offsets, weights, n_chunks, &b, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(d_order, h_order.data(), (size_t)m * 4, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(d_aoff, h_aoff.data(), (size_t)(m + 1) * 8, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess && n_caps > 0)
    e = cudaMemcpyAsync(d_caps, capacities, (size_t)n_caps * 8, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(d_costs, 0, (size_t)(n_caps > 0 ? n_caps : 1) * 8, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(compulsory, 0, 8, st);
  if (e == cudaSuccess) e = run_lex(s, &b, bits_for((uint64_t)n_chunks), true, st, &launches);
  if (e == cudaSuccess && N > 0) {
    for (int k = 1; k < K; ++k) k_sparse_level<<<grid_for(m), kThreads, 0, st>>>(b.lcp, m, k);
    k_new_nodes<<<grid_for(m), kThreads, 0, st>>>(b.ord, m, b.off, b.lcp, node_base);
    launches += K;
    e = exclusive_scan(node_base, m, as.sums, st, &launches);
    if (e == cudaSuccess) {
      k_accesses<<<grid_for(m), kThreads, 0, st>>>(d_order, m, b.off, b.chunk, b.w, b.lexpos, b.lcp, K, node_base,
                                                   d_aoff, node, acc_id, aw, asuf, aowner);
      ++launches;
      uint32_t* keys = node;
      uint32_t* vals = acc_id;
      e = radix_sort(&keys, &vals, as, N, bits_for((uint64_t)N), st, &launches);
      if (e == cudaSuccess) {
        k_prev_next<<<grid_for(N), kThreads, 0, st>>>(keys, vals, N, aowner, prev_t, next_t);
        k_scan_limit<<<1, 32, 0, st>>>(d_caps, n_caps, b.trie, limit);
        k_distance<<<grid_for(m * 32, 64), kDistThreads, 0, st>>>(m, d_aoff, prev_t, next_t, aw, asuf, limit,
                                                                         dist);
        k_cache_costs<<<grid_for(N, 8), kThreads, 0, st>>>(dist, aw, N, d_caps, n_caps, d_costs, compulsory);
        launches += 4;
        e = cudaGetLastError();
      }
    }
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(&h_trie, b.trie, 8, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&h_first, compulsory, 8, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess && n_caps > 0)
    e = cudaMemcpyAsync(h_costs.data(), d_costs, (size_t)n_caps * 8, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(mem);
  if (e != cudaSuccess) return cuda_status(e);
  // every trie node is first touched exactly once
  if (h_first != h_trie) return MPT_ERR_INTERNAL;
  for (int32_t i = 0; i < n_caps; ++i) costs[i] = (int64_t)h_costs[(size_t)i];
  if (unbounded) *unbounded = (int64_t)h_trie;
  return MPT_OK;
}

mpt_status mpt_layout_pinned(const int64_t* weights, int64_t n_chunks, int32_t m, const int64_t* ranked_offsets,
                             const int64_t* ranked_chunks, int32_t t, int32_t method, void* stream,
                             int64_t* perm_chunks, int32_t* serve_order, int64_t* cost) {
  using namespace mpt;
  if (!weights || !ranked_offsets || n_chunks < 1 || n_chunks >= INT32_MAX || m < 1 || t < 0) return MPT_ERR_INVALID_ARG;
  if (method != MPT_PIN_EXACT && method != MPT_PIN_GREEDY) return MPT_ERR_INVALID_ARG;
  if (method == MPT_PIN_EXACT && m > 32) return MPT_ERR_TOO_LARGE;
  if (ranked_offsets[0] != 0) return MPT_ERR_INVALID_ARG;
  const int64_t total = ranked_offsets[m];
  if (total > 0 && !ranked_chunks) return MPT_ERR_INVALID_ARG;
  for (int32_t i = 0; i < m; ++i)
    if (ranked_offsets[i + 1] < ranked_offsets[i]) return MPT_ERR_INVALID_ARG;
  for (int64_t p = 0; p < total; ++p)
    if (ranked_chunks[p] < 0 || ranked_chunks[p] >= n_chunks) return MPT_ERR_INVALID_ARG;
  // free part of request i: its ranked list after the first t entries
  std::vector<int64_t> foff((size_t)m + 1, 0), fchunks, seq((size_t)(total > 0 ? total : 1));
  for (int32_t i = 0; i < m; ++i) {
    const int64_t a = ranked_offsets[i], b = ranked_offsets[i + 1];
    const int64_t pin = b - a < t ? b - a : t;
    for (int64_t p = a + pin; p < b; ++p) fchunks.push_back(ranked_chunks[p]);
    foff[(size_t)i + 1] = (int64_t)fchunks.size();
  }
  std::vector<int64_t> fperm(fchunks.size() > 0 ? fchunks.size() : 1);
  mpt_status ms;
  if (method == MPT_PIN_EXACT) {
    const int64_t words = (n_chunks + 63) / 64;
    std::vector<uint64_t> bits((size_t)m * (size_t)words, 0);
    for (int32_t i = 0; i < m; ++i)
      for (int64_t p = foff[(size_t)i]; p < foff[(size_t)i + 1]; ++p) {
        const int64_t x = fchunks[(size_t)p];
        uint64_t& wd = bits[(size_t)i * (size_t)words + (size_t)(x >> 6)];
        if (wd >> (x & 63) & 1ull) return MPT_ERR_INVALID_ARG;  // repeated chunk
        wd |= 1ull << (x & 63);
      }
    mpt_ctx* ctx = nullptr;
    if ((ms = mpt_create(weights, n_chunks, bits.data(), m, &ctx)) != MPT_OK) return ms;
    int64_t opt = 0;
    std::vector<int64_t> poff((size_t)m + 1);
    ms = mpt_solve(ctx, nullptr, 0, stream, &opt);
    if (ms == MPT_OK) ms = mpt_layout(ctx, poff.data(), fperm.data(), nullptr);
    mpt_destroy(ctx);
    if (ms != MPT_OK) return ms;
    // mpt_layout's request ranges coincide with the free CSR (same sizes)
    for (int32_t i = 0; i <= m; ++i)
      if (poff[(size_t)i] != foff[(size_t)i]) return MPT_ERR_INTERNAL;
  } else {
    ms = mpt_greedy(weights, n_chunks, m, foff.data(), fchunks.empty() ? nullptr : fchunks.data(), stream, nullptr,
                    nullptr, nullptr, nullptr, nullptr, fperm.data(), nullptr);
    if (ms != MPT_OK) return ms;
  }
  // strings: free layout, then the pinned passages in relevance order
  for (int32_t i = 0; i < m; ++i) {
    const int64_t a = ranked_offsets[i], b = ranked_offsets[i + 1];
    const int64_t pin = b - a < t ? b - a : t;
    int64_t o = a;
    for (int64_t p = foff[(size_t)i]; p < foff[(size_t)i + 1]; ++p) seq[(size_t)o++] = fperm[(size_t)p];
    for (int64_t p = a; p < a + pin; ++p) seq[(size_t)o++] = ranked_chunks[p];
  }
  if (perm_chunks && total > 0) std::memcpy(perm_chunks, seq.data(), (size_t)total * 8);
  if (serve_order) {
    ms = mpt_serve_order(n_chunks, m, ranked_offsets, seq.data(), nullptr, 0, stream, serve_order);
    if (ms != MPT_OK) return ms;
  }
  if (cost) {
    ms = trie_cost_lex(weights, n_chunks, m, ranked_offsets, seq.data(), reinterpret_cast<cudaStream_t>(stream), cost);
    if (ms != MPT_OK) return ms;
  }
  return MPT_OK;
}

}  // extern "C"
