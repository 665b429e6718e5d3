// Batched exact solve of many small instances (m <= 13 requests each), one
// block per instance with every table in shared memory.
//
// This is the paper's own use of the exact recurrence (Sec. 6.2: 72 synthetic
// groups of 10-15 requests; Sec. 7: real request groups of at most 13): many
// independent groups, each small enough that its 2^m tables fit on chip.
// Per block, in order:
//   1. gather the instance's (chunk, request) occurrences and sort them by
//      chunk id (bitonic sort), so that each distinct chunk x gets its
//      request set N_x (S_x of Sec. 3) by OR-ing its run;
//   2. g(T) = sum of w(x) over N_x = T, then superset sums: wI(S) = w(I(S));
//   3. the Sec. 3.1 recurrence layer by layer, F(S) = min over splits of
//      F(A) + F(S \ A) - wI(S), the split named by its part A holding the
//      lowest request of S and the smallest such A kept on ties;
//   4. the hierarchy walk of the Thm 1 proof: request i's chunks ordered by
//      (depth of the highest node on its path inside N_x, chunk id), and the
//      left-to-right leaf order (Thm 7).
// Values are kept in 32 bits: the host accepts an instance only when
// sum_i w(R_i) < 2^31, so every F and every split sum fits.
#include "mpt_internal.cuh"

namespace mpt {
namespace {

constexpr int kBatchThreads = 256;

__device__ __forceinline__ int block_exclusive_scan(int v, int* tmp) {
  // tmp: kBatchThreads ints of shared memory
  const int t = threadIdx.x;
  tmp[t] = v;
  __syncthreads();
  for (int off = 1; off < kBatchThreads; off <<= 1) {
    const int add = t >= off ? tmp[t - off] : 0;
    __syncthreads();
    tmp[t] += add;
    __syncthreads();
  }
  const int incl = tmp[t];
  __syncthreads();
  return incl - v;
}

__global__ void __launch_bounds__(kBatchThreads)
k_batch_solve(const int64_t* __restrict__ weights, const int64_t* __restrict__ inst_req,
              const int64_t* __restrict__ req_off, const int64_t* __restrict__ chunks,
              const int64_t* __restrict__ tab_off, int occ_cap, int max_m, int64_t* __restrict__ opt_out,
              int64_t* __restrict__ F_out, uint32_t* __restrict__ split_out, int64_t* __restrict__ perm_out,
              int32_t* __restrict__ dfs_out, int32_t* __restrict__ status) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int inst = blockIdx.x;
  const int64_t r0 = inst_req[inst], r1 = inst_req[inst + 1];
  const int m = (int)(r1 - r0);
  const int64_t o0 = req_off[r0], o1 = req_off[r1];
  const int occ = (int)(o1 - o0);
  const int N = 1 << m;
  int P2 = 1;
  while (P2 < occ) P2 <<= 1;

  // shared layout (sized for max_m and occ_cap by the host)
  unsigned long long* keys = reinterpret_cast<unsigned long long*>(smem_raw);  // [occ_cap] sort keys, later walk keys
  uint32_t* wI = reinterpret_cast<uint32_t*>(keys + occ_cap);                  // [2^max_m]
  uint32_t* F = wI + (1 << max_m);                                              // [2^max_m]
  uint16_t* split = reinterpret_cast<uint16_t*>(F + (1 << max_m));             // [2^max_m]
  int32_t* cx = reinterpret_cast<int32_t*>(split + (1 << max_m));              // [occ_cap] distinct chunk ids
  uint32_t* cN = reinterpret_cast<uint32_t*>(cx + occ_cap);                    // [occ_cap] their request sets
  int* tmp = reinterpret_cast<int*>(cN + occ_cap);                              // [kBatchThreads]
  __shared__ uint32_t anc[16][16];
  __shared__ int leaf_depth[16], fill[16], dfs_s[16];
  __shared__ int ndistinct, bad;

  const int t = threadIdx.x;
  if (t == 0) {
    bad = 0;
    ndistinct = 0;
  }
  // 1. occurrences -> sort keys (chunk id << 4 | request), padding at the end
  for (int j = t; j < P2; j += kBatchThreads) keys[j] = ~0ull;
  __syncthreads();
  for (int i = 0; i < m; ++i) {
    const int64_t a = req_off[r0 + i] - o0, b = req_off[r0 + i + 1] - o0;
    for (int64_t j = a + t; j < b; j += kBatchThreads)
      keys[j] = ((unsigned long long)chunks[o0 + j] << 4) | (unsigned long long)i;
  }
  __syncthreads();
  for (int size = 2; size <= P2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int j = t; j < P2; j += kBatchThreads) {
        const int p = j ^ stride;
        if (p > j) {
          const bool up = (j & size) == 0;
          const unsigned long long a = keys[j], b = keys[p];
          if ((a > b) == up) {
            keys[j] = b;
            keys[p] = a;
          }
        }
      }
      __syncthreads();
    }
  }
  // distinct chunks: run starts, their ranks, and request sets
  for (int base = 0; base < occ; base += kBatchThreads) {
    const int j = base + t;
    const bool start = j < occ && (j == 0 || (keys[j] >> 4) != (keys[j - 1] >> 4));
    const int rank = block_exclusive_scan(start ? 1 : 0, tmp);
    const int before = ndistinct;
    __syncthreads();
    if (start) {
      cx[before + rank] = (int32_t)(keys[j] >> 4);
      cN[before + rank] = 0;
    }
    if (t == kBatchThreads - 1) ndistinct = before + rank + (start ? 1 : 0);
    __syncthreads();
  }
  // request bits: each occurrence ORs its request into its chunk's run
  for (int j = t; j < occ; j += kBatchThreads) {
    // the run of occurrence j is the number of run starts at or before j, minus one
    int lo = 0, hi = ndistinct - 1;
    const int32_t x = (int32_t)(keys[j] >> 4);
    while (lo < hi) {  // cx is increasing: find the entry equal to x
      const int mid = (lo + hi) >> 1;
      if (cx[mid] < x) lo = mid + 1; else hi = mid;
    }
    atomicOr(&cN[lo], 1u << (keys[j] & 15ull));
  }
  for (int S = t; S < N; S += kBatchThreads) wI[S] = 0;
  __syncthreads();
  const int nd = ndistinct;

  // 2. g(T), then superset sums over the m request bits
  for (int u = t; u < nd; u += kBatchThreads) atomicAdd(&wI[cN[u]], (uint32_t)weights[cx[u]]);
  __syncthreads();
  for (int j = 0; j < m; ++j) {
    for (int p = t; p < (N >> 1); p += kBatchThreads) {
      const int S = ((p >> j) << (j + 1)) | (p & ((1 << j) - 1));
      wI[S] += wI[S | (1 << j)];
    }
    __syncthreads();
  }

  // 3. the recurrence, one popcount layer at a time
  for (int S = t; S < N; S += kBatchThreads) {
    if ((S & (S - 1)) == 0) {
      F[S] = S ? wI[S] : 0u;
      split[S] = 0;
    }
  }
  __syncthreads();
  for (int k = 2; k <= m; ++k) {
    const int count = (int)c_binom.v[m][k];
    // lanes per subset: enough to keep the block busy, at most 32
    int g = 0;
    while ((count << (g + 1)) <= kBatchThreads && g < 5 && g < k - 1) ++g;
    const int G = 1 << g;
    const int per_pass = kBatchThreads >> g;
    for (int base = 0; base < count; base += per_pass) {
      const int idx = base + (t >> g);
      const uint32_t r = (uint32_t)t & (uint32_t)(G - 1);
      unsigned long long best = ~0ull;
      uint32_t S = 0;
      if (idx < count) {
        S = colex_unrank((unsigned long long)idx, k, m);
        const uint32_t low = S & (~S + 1u);
        const uint32_t rest = S ^ low;
        uint32_t hi = 0, rr = rest;
        for (int q = 0; q < g; ++q) {
          const uint32_t top = 1u << (31 - __clz(rr));
          hi |= top;
          rr ^= top;
        }
        const uint32_t freem = rest ^ hi;
        const uint32_t fixed = deposit_bits(r, hi);
        uint32_t sub = 0;
        do {
          const uint32_t part = fixed | sub;
          if (part != rest) {
            const uint32_t A = low | part;
            const unsigned long long c = ((unsigned long long)(F[A] + F[S ^ A]) << 16) | A;
            best = c < best ? c : best;
          }
          sub = (sub - freem) & freem;
        } while (sub != 0);
      }
      for (int off = G >> 1; off > 0; off >>= 1) {
        const unsigned long long o = __shfl_xor_sync(0xFFFFFFFFu, best, off);
        best = o < best ? o : best;
      }
      if (idx < count && r == 0) {
        F[S] = (uint32_t)(best >> 16) - wI[S];
        split[S] = (uint16_t)(best & 0xFFFFu);
      }
    }
    __syncthreads();
  }

  // outputs: tables and OPT
  const int64_t tb = tab_off[inst];
  for (int S = t; S < N; S += kBatchThreads) {
    F_out[tb + S] = (int64_t)F[S];
    split_out[tb + S] = split[S];
  }
  if (t == 0) opt_out[inst] = (int64_t)F[N - 1];

  // 4. hierarchy walk
  if (t < 16) {

    fill[t] = 0;
    leaf_depth[t] = 0;
  }
  if (t == 0) {
    uint32_t stk[32];
    int stk_d[32];
    int sp = 0, nleaf = 0;
    stk[sp] = (uint32_t)N - 1u;
    stk_d[sp] = 0;
    ++sp;
    while (sp > 0 && !bad) {
      --sp;
      const uint32_t S = stk[sp];
      const int d = stk_d[sp];
      for (uint32_t rr = S; rr; rr &= rr - 1) anc[__ffs(rr) - 1][d] = S;
      if ((S & (S - 1)) == 0) {
        const int i = __ffs(S) - 1;
        leaf_depth[i] = d;
        dfs_s[nleaf++] = i;
        continue;
      }
      const uint32_t A = split[S];
      if (A == 0 || (A & ~S) != 0 || A == S || sp + 2 > 32) {
        bad = 1;
        break;
      }
      stk[sp] = S ^ A;
      stk_d[sp] = d + 1;
      ++sp;
      stk[sp] = A;
      stk_d[sp] = d + 1;
      ++sp;
    }
  }
  __syncthreads();
  if (bad) {
    if (t == 0) status[inst] = 1;
    return;
  }
  if (t < m) dfs_out[r0 + t] = dfs_s[t];
  // keys (depth, chunk id) into each request's own slot range, then rank them
  for (int u = t; u < nd; u += kBatchThreads) {
    const uint32_t Nx = cN[u];
    for (uint32_t rr = Nx; rr; rr &= rr - 1) {
      const int i = __ffs(rr) - 1;
      int d = 0;
      while (d < leaf_depth[i] && (anc[i][d] & ~Nx) != 0) ++d;
      const int slot = atomicAdd(&fill[i], 1);
      const int64_t base = req_off[r0 + i] - o0;
      keys[base + slot] = ((unsigned long long)d << 32) | (unsigned long long)(uint32_t)cx[u];
    }
  }
  __syncthreads();
  const int lane = t & 31, warp = t >> 5;
  for (int i = warp; i < m; i += kBatchThreads / 32) {
    const int64_t base = req_off[r0 + i] - o0;
    const int len = (int)(req_off[r0 + i + 1] - req_off[r0 + i]);
    for (int j = lane; j < len; j += 32) {
      const unsigned long long kj = keys[base + j];
      int rank = 0;
      for (int q = 0; q < len; ++q) rank += keys[base + q] < kj;
      perm_out[o0 + base + rank] = (int64_t)(kj & 0xFFFFFFFFull);
    }
  }
  if (t == 0) status[inst] = 0;
}

}  // namespace

size_t batch_smem_bytes(int max_m, int occ_cap) {
  return (size_t)occ_cap * 8 + ((size_t)4 << max_m) * 2 + ((size_t)2 << max_m) + (size_t)occ_cap * 8 +
         (size_t)kBatchThreads * 4 + 64;
}

cudaError_t launch_batch(int batch, int max_m, int occ_cap, const int64_t* weights, const int64_t* inst_req,
                         const int64_t* req_off, const int64_t* chunks, const int64_t* tab_off, int64_t* opt,
                         int64_t* F, uint32_t* split, int64_t* perm, int32_t* dfs, int32_t* status,
                         cudaStream_t stream) {
  const size_t smem = batch_smem_bytes(max_m, occ_cap);
  cudaError_t e = cudaFuncSetAttribute(k_batch_solve, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_batch_solve<<<(unsigned)batch, kBatchThreads, smem, stream>>>(weights, inst_req, req_off, chunks, tab_off, occ_cap,
                                                                  max_m, opt, F, split, perm, dfs, status);
  return cudaGetLastError();
}

}  // namespace mpt
