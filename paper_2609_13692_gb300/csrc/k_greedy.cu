// Agglomerative common-intersection hierarchy (Sec. 6.2; H_g of Thm 6) and
// the spanning-tree lower bound (Sec. 6.3), for request counts far beyond the
// exact recurrence (m up to 16384).
//
// Greedy: every request starts as a cluster with signature R_i; the two active
// clusters with the heaviest common signature w(I(A) cap I(B)) merge, the
// merged signature being that intersection.  A cluster lives in the slot of
// its smallest request; ties go to the smallest slot pair (a, b), a < b, and
// the merged cluster keeps slot a.  The layout walks the hierarchy as in the
// Thm 1 proof.  Lower bound: sum_i w(R_i) - MaxSpanningTree(w(R_i cap R_j)).
//
// Kernels: k_pair_weights fills W[i][j] = w(R_i cap R_j) (sorted chunk lists,
// merge-intersection); Borůvka rounds find the maximum spanning tree of W;
// k_greedy_merge runs all m - 1 merges in one block, keeping for every active
// slot an upper bound on its best partner as a 64-bit key (weight, then the
// smallest slot pair) and rescanning a row only when its key is found stale; k_greedy_layout climbs each
// (request, chunk) occurrence to the highest node whose signature still holds
// the chunk, and ranks each request's chunks by (depth, chunk id).
#include "../../include/mpt.h"
#include "mpt_internal.cuh"

#include <algorithm>
#include <vector>

namespace mpt {
namespace {

constexpr int kSigMax = 128;       // longest request accepted
constexpr int kMaxGreedyM = 16384;  // slot ids fit in 14 bits
constexpr int kGreedyThreads = 1024;

__device__ __forceinline__ uint32_t sig_weight(const int32_t* a, int la, const int32_t* b, int lb,
                                               const int64_t* __restrict__ w) {
  uint32_t s = 0;
  int i = 0, j = 0;
  while (i < la && j < lb) {
    const int32_t x = a[i], y = b[j];
    if (x == y) {
      s += (uint32_t)w[x];
      ++i;
      ++j;
    } else if (x < y) {
      ++i;
    } else {
      ++j;
    }
  }
  return s;
}

// key of pair {d, e} with common weight v: larger is better (weight, then the
// smaller slot pair)
__device__ __forceinline__ unsigned long long pair_key(uint32_t d, uint32_t e, uint32_t v) {
  const uint32_t a = min(d, e), b = max(d, e);
  return ((unsigned long long)v << 28) | (unsigned long long)((1u << 28) - 1u - ((a << 14) | b));
}
__device__ __forceinline__ void key_pair(unsigned long long k, uint32_t* a, uint32_t* b) {
  const uint32_t p = (1u << 28) - 1u - (uint32_t)(k & ((1u << 28) - 1u));
  *a = p >> 14;
  *b = p & ((1u << 14) - 1u);
}

__global__ void k_pair_weights(int m, const int32_t* __restrict__ sig, const int32_t* __restrict__ len,
                               const int64_t* __restrict__ w, uint32_t* __restrict__ W) {
  const int i = blockIdx.y;
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < m; j += gridDim.x * blockDim.x) {
    if (j < i) continue;
    const uint32_t v = (j == i) ? 0u : sig_weight(sig + (size_t)i * kSigMax, len[i], sig + (size_t)j * kSigMax, len[j], w);
    W[(size_t)i * m + j] = v;
    W[(size_t)j * m + i] = v;
  }
}

// best partner of every slot: warp per row
__global__ void k_row_best(int m, const uint32_t* __restrict__ W, unsigned long long* __restrict__ best) {
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  for (int d = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; d < m; d += warps) {
    unsigned long long b = 0;
    for (int e = lane; e < m; e += 32)
      if (e != d) b = max(b, pair_key((uint32_t)d, (uint32_t)e, W[(size_t)d * m + e]));
    for (int off = 16; off > 0; off >>= 1) b = max(b, __shfl_xor_sync(0xFFFFFFFFu, b, off));
    if (lane == 0) best[d] = b;
  }
}

__device__ unsigned long long block_max_u64(unsigned long long v, unsigned long long* red) {
  for (int off = 16; off > 0; off >>= 1) v = max(v, __shfl_xor_sync(0xFFFFFFFFu, v, off));
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < (int)(blockDim.x >> 5) ? red[lane] : 0ull;
    for (int off = 16; off > 0; off >>= 1) v = max(v, __shfl_xor_sync(0xFFFFFFFFu, v, off));
    if (lane == 0) red[32] = v;
  }
  __syncthreads();
  const unsigned long long r = red[32];
  __syncthreads();
  return r;
}

// Maximum spanning tree of W (Borůvka).  Edges are ordered by pair_key
// (weight, then the smaller slot pair), so every edge key is distinct and the
// tree is unique; its weight is the maximum spanning-tree weight (Sec. 6.3).
// A round: each vertex's heaviest edge to another component (warp per row),
// each component's heaviest (atomicMax), components hook along them (a pair
// of components that chose the same edge keeps the smaller id as root, and
// that edge is counted once), then every vertex jumps to its root.  Every
// round at least halves the number of components.
__global__ void k_bv_vertex_best(int m, const uint32_t* __restrict__ W, const int32_t* __restrict__ comp,
                                 unsigned long long* __restrict__ cbest) {
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  for (int v = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; v < m; v += warps) {
    const int cv = comp[v];
    unsigned long long b = 0;
    for (int u = lane; u < m; u += 32)
      if (comp[u] != cv) b = max(b, pair_key((uint32_t)v, (uint32_t)u, W[(size_t)v * m + u]));
    for (int off = 16; off > 0; off >>= 1) b = max(b, __shfl_xor_sync(0xFFFFFFFFu, b, off));
    if (lane == 0 && b) atomicMax(&cbest[cv], b);
  }
}

__global__ void k_bv_hook(int m, const int32_t* __restrict__ comp, const unsigned long long* __restrict__ cbest,
                          int32_t* __restrict__ parent, unsigned long long* __restrict__ total) {
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < m; c += gridDim.x * blockDim.x) {
    if (comp[c] != c) continue;  // not a component root
    const unsigned long long k = cbest[c];
    if (k == 0) {
      parent[c] = c;
      continue;
    }
    uint32_t a, b;
    key_pair(k, &a, &b);
    const int o = comp[a] == c ? comp[b] : comp[a];
    const bool mutual = cbest[o] == k;
    parent[c] = (mutual && c < o) ? c : o;
    if (!(mutual && o < c)) atomicAdd(total, k >> 28);
  }
}

__global__ void k_bv_jump(int m, int32_t* __restrict__ comp, const int32_t* __restrict__ parent) {
  for (int v = blockIdx.x * blockDim.x + threadIdx.x; v < m; v += gridDim.x * blockDim.x) {
    int r = comp[v];
    for (int step = 0; step < m && parent[r] != r; ++step) r = parent[r];
    comp[v] = r;
  }
}

__global__ void k_bv_reset(int m, unsigned long long* __restrict__ cbest) {
  for (int v = blockIdx.x * blockDim.x + threadIdx.x; v < m; v += gridDim.x * blockDim.x) cbest[v] = 0;
}

__global__ void k_iota32(int m, int32_t* __restrict__ a) {
  for (int v = blockIdx.x * blockDim.x + threadIdx.x; v < m; v += gridDim.x * blockDim.x) a[v] = v;
}


// All m - 1 merges (one block).  best[d] is an upper bound on row d's best
// pair key: pair weights only decrease as clusters merge, so a key stays an
// upper bound until its row is rescanned.  The largest bound is merged only
// if it is still exact (both slots active, weight unchanged); otherwise its
// rows are rescanned and the choice is repeated.  Every rescan makes a row
// exact, so a step repeats at most m times (kept as a hard cap).
// Weight of sig_d (sorted, in global memory) within the merged signature
// s_new (sorted, shared memory): binary search of each chunk of sig_d.
__device__ __forceinline__ uint32_t sig_weight_in(const int32_t* __restrict__ sd, int ld, const int32_t* s_new,
                                                  int ln, const int64_t* __restrict__ w) {
  uint32_t s = 0;
  for (int q = 0; q < ld; ++q) {
    const int32_t x = sd[q];
    int lo = 0, hi = ln;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (s_new[mid] < x) lo = mid + 1; else hi = mid;
    }
    if (lo < ln && s_new[lo] == x) s += (uint32_t)w[x];
  }
  return s;
}


// All m - 1 merges in one block, with lazy best keys: sb[d] (shared memory)
// is an upper bound on slot d's best pair key (weights only decrease as
// signatures shrink), 0 once d is merged away, and gmax[g] is the largest of
// sb[32 g .. 32 g + 31].  The largest key is merged only if it is still
// exact; otherwise the rows of its two slots are rescanned and the search
// repeats.
constexpr int kMaxGroups = kMaxGreedyM / 32;

__device__ __forceinline__ void refresh_group(int m, int g, const unsigned long long* sb, unsigned long long* gmax) {
  if (threadIdx.x < 32) {
    const int d = g * 32 + (int)threadIdx.x;
    unsigned long long v = d < m ? sb[d] : 0ull;
    for (int off = 16; off > 0; off >>= 1) v = max(v, __shfl_xor_sync(0xFFFFFFFFu, v, off));
    if (threadIdx.x == 0) gmax[g] = v;
  }
}

__device__ unsigned long long smem_row_best(int m, int d, const uint32_t* __restrict__ W, const uint8_t* act,
                                            unsigned long long* red) {
  unsigned long long bb = 0;
  const uint32_t* row = W + (size_t)d * m;
  for (int e = threadIdx.x; e < m; e += blockDim.x)
    if (e != d && act[e]) bb = max(bb, pair_key((uint32_t)d, (uint32_t)e, row[e]));
  return block_max_u64(bb, red);
}

__global__ void __launch_bounds__(kGreedyThreads)
k_greedy_merge(int m, const int64_t* __restrict__ w, int32_t* __restrict__ sig, int32_t* __restrict__ len,
               uint32_t* __restrict__ W, const unsigned long long* __restrict__ best0, int32_t* __restrict__ node,
               int32_t* __restrict__ merges, int64_t* __restrict__ values, int32_t* __restrict__ children,
               int32_t* __restrict__ node_sig, int32_t* __restrict__ node_len, int32_t* __restrict__ error) {
  extern __shared__ __align__(16) unsigned char gsm[];
  unsigned long long* sb = reinterpret_cast<unsigned long long*>(gsm);        // [m]
  unsigned long long* gmax = sb + m;                                          // [ceil(m / 32)]
  uint8_t* act = reinterpret_cast<uint8_t*>(gmax + kMaxGroups);               // [m]
  __shared__ unsigned long long red[33];
  __shared__ int32_t s_a[kSigMax], s_b[kSigMax], s_new[kSigMax];
  __shared__ int s_len;
  __shared__ int warp_cnt[kGreedyThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int groups = (m + 31) / 32;
  for (int d = threadIdx.x; d < m; d += blockDim.x) {
    act[d] = 1;
    node[d] = d;
    sb[d] = best0[d];
  }
  __syncthreads();
  for (int g = warp; g < groups; g += kGreedyThreads / 32) {
    const int d = g * 32 + lane;
    unsigned long long v = d < m ? sb[d] : 0ull;
    for (int off = 16; off > 0; off >>= 1) v = max(v, __shfl_xor_sync(0xFFFFFFFFu, v, off));
    if (lane == 0) gmax[g] = v;
  }
  __syncthreads();
  for (int t = 0; t < m - 1; ++t) {
    uint32_t a = 0, b = 0, v = 0;
    int tries = 0;
    for (;;) {
      const unsigned long long c = (int)threadIdx.x < groups ? gmax[threadIdx.x] : 0ull;
      const unsigned long long top = block_max_u64(c, red);
      key_pair(top, &a, &b);
      v = (uint32_t)(top >> 28);
      if (top != 0 && act[a] && act[b] && W[(size_t)a * m + b] == v) break;
      if (top == 0 || ++tries > m + 1) {
        if (threadIdx.x == 0) atomicOr(error, 1);
        return;
      }
      if (act[a]) {
        const unsigned long long r = smem_row_best(m, (int)a, W, act, red);
        if (threadIdx.x == 0) sb[a] = r;
        __syncthreads();
        refresh_group(m, (int)a >> 5, sb, gmax);
      }
      if (act[b]) {
        const unsigned long long r = smem_row_best(m, (int)b, W, act, red);
        if (threadIdx.x == 0) sb[b] = r;
        __syncthreads();
        refresh_group(m, (int)b >> 5, sb, gmax);
      }
      __syncthreads();
    }
    // merged signature: the chunks of a that b holds, in order
    const int la = len[a], lb = len[b];
    for (int q = threadIdx.x; q < la; q += blockDim.x) s_a[q] = sig[(size_t)a * kSigMax + q];
    for (int q = threadIdx.x; q < lb; q += blockDim.x) s_b[q] = sig[(size_t)b * kSigMax + q];
    __syncthreads();
    bool keep = false;
    int32_t x = 0;
    if ((int)threadIdx.x < la) {
      x = s_a[threadIdx.x];
      int lo = 0, hi = lb;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (s_b[mid] < x) lo = mid + 1; else hi = mid;
      }
      keep = lo < lb && s_b[lo] == x;
    }
    const unsigned bal = __ballot_sync(0xFFFFFFFFu, keep);
    if (lane == 0) warp_cnt[warp] = __popc(bal);
    __syncthreads();
    if (keep) {
      int before = __popc(bal & ((1u << lane) - 1u));
      for (int q = 0; q < warp; ++q) before += warp_cnt[q];  // kSigMax <= 128: at most four warps
      s_new[before] = x;
    }
    if (threadIdx.x == 0) {
      int n = 0;
      for (int q = 0; q < (kSigMax + 31) / 32; ++q) n += warp_cnt[q];
      s_len = n;
      merges[2 * t] = (int32_t)a;
      merges[2 * t + 1] = (int32_t)b;
      values[t] = v;
      children[2 * t] = node[a];
      children[2 * t + 1] = node[b];
    }
    __syncthreads();
    const int ln = s_len;
    for (int q = threadIdx.x; q < ln; q += blockDim.x) {
      sig[(size_t)a * kSigMax + q] = s_new[q];
      node_sig[(size_t)t * kSigMax + q] = s_new[q];
    }
    // new pair weights of the merged slot: zero wherever either old weight was
    // zero (the merged signature is a subset of both)
    for (int d = threadIdx.x; d < m; d += blockDim.x) {
      if (!act[d] || d == (int)a || d == (int)b) continue;
      const uint32_t wa = W[(size_t)a * m + d], wb = W[(size_t)b * m + d];
      const uint32_t wv = (wa == 0 || wb == 0 || ln == 0)
                              ? 0u
                              : sig_weight_in(sig + (size_t)d * kSigMax, len[d], s_new, ln, w);
      W[(size_t)a * m + d] = wv;
      W[(size_t)d * m + a] = wv;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      len[a] = ln;
      node_len[t] = ln;
      node[a] = m + t;
      act[b] = 0;
      sb[b] = 0;
    }
    __syncthreads();
    const unsigned long long r = smem_row_best(m, (int)a, W, act, red);
    if (threadIdx.x == 0) sb[a] = r;
    __syncthreads();
    refresh_group(m, (int)a >> 5, sb, gmax);
    __syncthreads();
    refresh_group(m, (int)b >> 5, sb, gmax);
    __syncthreads();
  }
}

size_t merge_smem_bytes(int m) { return (size_t)m * 8 + (size_t)kMaxGroups * 8 + (size_t)m + 16; }

// Parent and depth of every tree node and the left-to-right leaf order (one thread).
__global__ void k_greedy_tree(int m, const int32_t* __restrict__ children, int32_t* __restrict__ parent,
                              int32_t* __restrict__ depth, int32_t* __restrict__ stack, int32_t* __restrict__ dfs) {
  const int root = m == 1 ? 0 : 2 * m - 2;
  parent[root] = -1;
  depth[root] = 0;
  for (int t = m - 2; t >= 0; --t) {
    const int v = m + t;
    for (int c = 0; c < 2; ++c) {
      const int ch = children[2 * t + c];
      parent[ch] = v;
      depth[ch] = depth[v] + 1;
    }
  }
  int sp = 0, nl = 0;
  stack[sp++] = root;
  while (sp > 0) {
    const int v = stack[--sp];
    if (v < m) {
      dfs[nl++] = v;
      continue;
    }
    const int t = v - m;
    stack[sp++] = children[2 * t + 1];  // right after left
    stack[sp++] = children[2 * t];
  }
}

// Emission depth of every (request, chunk) occurrence: climb from the leaf
// while the parent's signature still holds the chunk.
__global__ void k_greedy_emit(int m, const int32_t* __restrict__ node_sig, const int32_t* __restrict__ node_len,
                              const int64_t* __restrict__ req_off, const int64_t* __restrict__ chunks,
                              const int32_t* __restrict__ parent, const int32_t* __restrict__ depth,
                              unsigned long long* __restrict__ keys) {
  const int64_t occ = req_off[m];
  for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < occ; j += (int64_t)gridDim.x * blockDim.x) {
    int lo = 0, hi = m - 1;  // request of occurrence j: the last i with req_off[i] <= j
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (req_off[mid] <= j) lo = mid; else hi = mid - 1;
    }
    const int32_t x = (int32_t)chunks[j];
    int v = lo;
    for (;;) {
      const int p = parent[v];
      if (p < 0) break;
      const int t = p - m;
      const int32_t* s = node_sig + (size_t)t * kSigMax;
      const int n = node_len[t];
      int a = 0, b = n;
      while (a < b) {
        const int mid = (a + b) >> 1;
        if (s[mid] < x) a = mid + 1; else b = mid;
      }
      if (a < n && s[a] == x) v = p; else break;
    }
    keys[j] = ((unsigned long long)depth[v] << 32) | (unsigned long long)(uint32_t)x;
  }
}

// Each request's chunks ranked by (emission depth, chunk id): warp per request.
__global__ void k_greedy_rank(int m, const int64_t* __restrict__ req_off, const unsigned long long* __restrict__ keys,
                              int64_t* __restrict__ perm) {
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  for (int i = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < m; i += warps) {
    const int64_t base = req_off[i];
    const int len = (int)(req_off[i + 1] - base);
    for (int q = lane; q < len; q += 32) {
      const unsigned long long kq = keys[base + q];
      int rank = 0;
      for (int r = 0; r < len; ++r) rank += keys[base + r] < kq;
      perm[base + rank] = (int64_t)(kq & 0xFFFFFFFFull);
    }
  }
}

}  // namespace
}  // namespace mpt

extern "C" mpt_status mpt_greedy(const int64_t* weights, int64_t n_chunks, int32_t m, const int64_t* req_offsets,
                                 const int64_t* chunk_ids, void* stream_ptr, int64_t* cost, int64_t* savings,
                                 int64_t* lower_bound, int32_t* merges, int64_t* merge_values, int64_t* perm_chunks,
                                 int32_t* dfs_order) {
  using namespace mpt;
  if (!weights || !req_offsets || n_chunks < 1 || n_chunks > INT32_MAX || m < 1) return MPT_ERR_INVALID_ARG;
  if (m > kMaxGreedyM) return MPT_ERR_TOO_LARGE;
  if (req_offsets[0] != 0) return MPT_ERR_INVALID_ARG;
  const int64_t occ = req_offsets[m];
  if (occ > 0 && !chunk_ids) return MPT_ERR_INVALID_ARG;
  for (int64_t x = 0; x < n_chunks; ++x)
    if (weights[x] <= 0) return MPT_ERR_INVALID_ARG;
  // sorted, de-duplicated-checked signatures; per-request weight < 2^32
  std::vector<int32_t> sig((size_t)m * kSigMax, 0), len((size_t)m, 0);
  int64_t total = 0;
  for (int i = 0; i < m; ++i) {
    const int64_t a = req_offsets[i], b = req_offsets[i + 1];
    if (b < a) return MPT_ERR_INVALID_ARG;
    if (b - a > kSigMax) return MPT_ERR_TOO_LARGE;
    std::vector<int64_t> ids(chunk_ids + a, chunk_ids + b);
    std::sort(ids.begin(), ids.end());
    int64_t rw = 0;
    for (size_t q = 0; q < ids.size(); ++q) {
      if (ids[q] < 0 || ids[q] >= n_chunks || (q > 0 && ids[q] == ids[q - 1])) return MPT_ERR_INVALID_ARG;
      sig[(size_t)i * kSigMax + q] = (int32_t)ids[q];
      rw += weights[ids[q]];
      if (rw >= ((int64_t)1 << 32)) return MPT_ERR_OVERFLOW;
    }
    len[(size_t)i] = (int32_t)ids.size();
    total += rw;
  }
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_ptr);
  // device buffers (this call allocates and frees its own)
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) & ~(size_t)255;
    return o;
  };
  const size_t M = (size_t)m;
  const size_t o_w = take((size_t)n_chunks * 8), o_sig = take(M * kSigMax * 4), o_len = take(M * 4),
               o_W = take(M * M * 4), o_best = take(M * 8), o_node = take(M * 4),
               o_re = take(M * 4 + 4), o_mer = take(M * 8), o_val = take(M * 8), o_ch = take(M * 8),
               o_nsig = take(M * kSigMax * 4), o_nlen = take(M * 4), o_roff = take((M + 1) * 8),
               o_chunks = take((size_t)std::max<int64_t>(occ, 1) * 8), o_par = take(2 * M * 4),
               o_dep = take(2 * M * 4), o_stk = take(2 * M * 4), o_keys = take((size_t)std::max<int64_t>(occ, 1) * 8),
               o_perm = take((size_t)std::max<int64_t>(occ, 1) * 8), o_dfs = take(M * 4), o_comp = take(M * 4),
               o_bpar = take(M * 4), o_cbest = take(M * 8), o_mst = take(8);
  char* d = nullptr;
  if (device_alloc(reinterpret_cast<void**>(&d), off) != cudaSuccess) return MPT_ERR_OUT_OF_MEMORY;
  const int64_t sms = sm_count();
  mpt_status st = MPT_OK;
  cudaError_t e = cudaSuccess;
  auto h2d = [&](size_t o, const void* h, size_t bytes) {
    if (e == cudaSuccess && bytes) e = cudaMemcpyAsync(d + o, h, bytes, cudaMemcpyHostToDevice, stream);
  };
  auto d2h = [&](void* h, size_t o, size_t bytes) {
    if (e == cudaSuccess && bytes && h) e = cudaMemcpyAsync(h, d + o, bytes, cudaMemcpyDeviceToHost, stream);
  };
  h2d(o_w, weights, (size_t)n_chunks * 8);
  h2d(o_sig, sig.data(), sig.size() * 4);
  h2d(o_len, len.data(), len.size() * 4);
  h2d(o_roff, req_offsets, (M + 1) * 8);
  h2d(o_chunks, chunk_ids, (size_t)occ * 8);
  if (e == cudaSuccess) e = cudaMemsetAsync(d + o_re, 0, 4, stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(d + o_mst, 0, 8, stream);
  auto I64 = [&](size_t o) { return reinterpret_cast<int64_t*>(d + o); };
  auto I32 = [&](size_t o) { return reinterpret_cast<int32_t*>(d + o); };
  auto U32 = [&](size_t o) { return reinterpret_cast<uint32_t*>(d + o); };
  auto U64 = [&](size_t o) { return reinterpret_cast<unsigned long long*>(d + o); };
  if (e == cudaSuccess) {
    dim3 grid((unsigned)((m + 255) / 256), (unsigned)m);
    k_pair_weights<<<grid, 256, 0, stream>>>(m, I32(o_sig), I32(o_len), I64(o_w), U32(o_W));
    {
      // maximum spanning tree by Borůvka rounds (each at least halves the components)
      const unsigned vb = (unsigned)std::min<int64_t>(((int64_t)m * 32 + 255) / 256, sms * 32);
      const unsigned eb = (unsigned)std::min<int64_t>((m + 255) / 256, sms * 8);
      k_iota32<<<eb, 256, 0, stream>>>(m, I32(o_comp));
      k_bv_reset<<<eb, 256, 0, stream>>>(m, U64(o_cbest));
      int rounds = 1;
      while ((1 << rounds) < m) ++rounds;
      for (int r = 0; r < rounds; ++r) {
        k_bv_vertex_best<<<vb, 256, 0, stream>>>(m, U32(o_W), I32(o_comp), U64(o_cbest));
        k_bv_hook<<<eb, 256, 0, stream>>>(m, I32(o_comp), U64(o_cbest), I32(o_bpar), U64(o_mst));
        k_bv_jump<<<eb, 256, 0, stream>>>(m, I32(o_comp), I32(o_bpar));
        k_bv_reset<<<eb, 256, 0, stream>>>(m, U64(o_cbest));
      }
    }
    k_row_best<<<(unsigned)((m * 32 + 255) / 256), 256, 0, stream>>>(m, U32(o_W), U64(o_best));
    {
      const size_t msm = merge_smem_bytes(m);
      e = cudaFuncSetAttribute(k_greedy_merge, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)msm);
      if (e == cudaSuccess)
        k_greedy_merge<<<1, kGreedyThreads, msm, stream>>>(m, I64(o_w), I32(o_sig), I32(o_len), U32(o_W), U64(o_best),
                                                           I32(o_node), I32(o_mer), I64(o_val), I32(o_ch), I32(o_nsig),
                                                           I32(o_nlen), I32(o_re));
    }
    k_greedy_tree<<<1, 1, 0, stream>>>(m, I32(o_ch), I32(o_par), I32(o_dep), I32(o_stk), I32(o_dfs));
    const int64_t eblocks = std::min<int64_t>((std::max<int64_t>(occ, 1) + 255) / 256, sms * 16);
    k_greedy_emit<<<(unsigned)eblocks, 256, 0, stream>>>(m, I32(o_nsig), I32(o_nlen), I64(o_roff), I64(o_chunks),
                                                         I32(o_par), I32(o_dep), U64(o_keys));
    k_greedy_rank<<<(unsigned)std::min<int64_t>(((int64_t)m * 32 + 255) / 256, sms * 16), 256, 0, stream>>>(
        m, I64(o_roff), U64(o_keys), I64(o_perm));
    e = cudaGetLastError();
  }
  std::vector<int64_t> vals(M > 1 ? M - 1 : 1, 0);
  unsigned long long mst = 0;
  int32_t flag = 0;
  d2h(&flag, o_re, 4);
  d2h(vals.data(), o_val, (M - 1) * 8);
  d2h(&mst, o_mst, 8);
  d2h(merges, o_mer, (M - 1) * 2 * 4);
  d2h(perm_chunks, o_perm, (size_t)occ * 8);
  d2h(dfs_order, o_dfs, M * 4);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) st = MPT_ERR_CUDA;
  else if (flag != 0) st = MPT_ERR_INTERNAL;
  cudaFree(d);
  if (st != MPT_OK) return st;
  int64_t sav = 0;
  for (size_t t = 0; t + 1 < M; ++t) sav += vals[t];
  if (merge_values && M > 1) std::copy(vals.begin(), vals.begin() + (M - 1), merge_values);
  if (savings) *savings = sav;
  if (cost) *cost = total - sav;
  if (lower_bound) *lower_bound = total - (int64_t)mst;
  return MPT_OK;
}
