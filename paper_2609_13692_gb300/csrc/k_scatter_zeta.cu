// K1: request-set scatter and K2: superset sums, giving w(I(S)) for every S
// (uint64 sums, or uint32 in the lean table when sum_i w(R_i) < 2^31).
//
// Sec. 3 defines S_x = {i : x in R_i}; here it is the m-bit mask N_x.  A chunk
// x lies in I(S) = intersection of R_i over i in S exactly when S is a subset
// of N_x, so
//     w(I(S)) = sum over T superset of S of g(T),   g(T) = sum of w(x) with N_x = T,
// which is the quantity w(I(B)) of the Sec. 3.1 recurrence.  K1 builds g and
// the list of chunks that some request uses; K2 is the superset-sum (zeta)
// transform over the 2^m table, done in shared-memory tiles so that each
// pass streams the table once with coalesced 128-byte rows.  For the blocked
// recurrence g is indexed in its rotated order (rot_index): the superset
// relation does not depend on the order of the index bits, so the same
// transform then yields w(I(S)) at the rotated position of S.
//
// Private chunks (blocked paths).  A chunk x with S_x = {i} is one maximal
// cluster of S_x in every hierarchy (t_x(H) = 1 in Thm 1), so it adds w(x)
// to F(S) for every S containing i whatever the splits: with
// pi_i = sum of w(x) over x with N_x = {i} and pi(S) = sum_{i in S} pi_i,
//     F(S) = F'(S) + pi(S),   F'({i}) = w(R_i) - pi_i,
//     F'(S) = min over splits of F'(A) + F'(B) - w(I(S))   (|S| >= 2),
// since pi(A) + pi(B) = pi(S) and w(I(S)) does not involve private chunks
// for |S| >= 2.  The argmin is the same.  Likewise a chunk that all m >= 2
// requests hold has S_x = the root, one cluster in every hierarchy: with u
// the weight of such chunks, F(S) = F'(S) + pi(S) + u for non-empty S, and
// the recurrence on F' sees w(I(S)) - u (u + u - u = u per split).  For the
// blocked paths K1 adds private chunks to pi_i and universal ones to u
// instead of to g, so the transform yields w(I(S)) - u for |S| >= 2 and
// w(R_i) - pi_i - u for S = {i}; the recurrence then runs on F', whose
// candidates stay below the shared weight sum_i (w(R_i) - pi_i - u), the
// quantity the packed keys must hold.
#include "mpt_internal.cuh"

namespace mpt {
namespace {

constexpr int kScatterThreads = 256;

// g is uint64 (int64 tables) or uint32 (lean tables, sum_i w(R_i) < 2^31).
// priv: pi_i of the private chunks and u of the universal ones (blocked
// paths, kOffsetSlots entries), or nullptr.
template <typename G>
__global__ void __launch_bounds__(kScatterThreads)
k_scatter(const int64_t* __restrict__ w, const uint64_t* __restrict__ bits, int64_t n, int m, int64_t words,
          G* __restrict__ g, unsigned long long* __restrict__ priv, uint32_t* __restrict__ used_N,
          int32_t* __restrict__ used_x, int32_t* __restrict__ counters, int64_t slots, bool rotated, int L, int b) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const uint32_t full = m >= 32 ? 0xFFFFFFFFu : (1u << m) - 1u;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < n; x += stride) {
    const int64_t word = x >> 6;
    const int sh = (int)(x & 63);
    uint32_t N = 0;
    for (int i = 0; i < m; ++i) N |= (uint32_t)((__ldg(&bits[(int64_t)i * words + word]) >> sh) & 1ull) << i;
    if (N) {
      if (priv && (N & (N - 1)) == 0)
        atomicAdd(&priv[__ffs(N) - 1], (unsigned long long)w[x]);
      else if (priv && N == full)  // m >= 2 here: for m = 1 the full set is a singleton
        atomicAdd(&priv[kUniversalSlot], (unsigned long long)w[x]);
      else if (!MPT_BAD(&counters[1], (rotated ? rot_index(N, L, b) : (size_t)N) < ((size_t)1 << m)))
        atomicAdd(&g[rotated ? rot_index(N, L, b) : (size_t)N], (G)w[x]);
      const int k = atomicAdd(&counters[0], 1);
      if (k < slots) {
        used_N[k] = N;
        used_x[k] = (int32_t)x;
      } else {
        atomicOr(&counters[1], kErrWorkspace);
      }
    }
  }
}

// Superset sums over the low `tb` index bits of each tile of 2^tb entries.
constexpr int kZetaLowBits = 12;
constexpr int kZetaThreads = 512;

template <typename G>
__global__ void __launch_bounds__(kZetaThreads) k_zeta_low(G* __restrict__ g, int tb, size_t n,
                                                           int32_t* __restrict__ flags) {
  __shared__ G t[1 << kZetaLowBits];
  const int size = 1 << tb;
  G* tile = g + ((size_t)blockIdx.x << tb);
  if (MPT_BAD(flags, ((size_t)blockIdx.x + 1) << tb <= n)) return;
  for (int i = threadIdx.x; i < size; i += blockDim.x) t[i] = tile[i];
  const int half = size >> 1;
  for (int j = 0; j < tb; ++j) {
    __syncthreads();
    const int lowmask = (1 << j) - 1;
    for (int p = threadIdx.x; p < half; p += blockDim.x) {
      const int i = ((p >> j) << (j + 1)) | (p & lowmask);  // bit j of i is 0
      t[i] += t[i | (1 << j)];
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < size; i += blockDim.x) tile[i] = t[i];
}

// The same for tb = 12 with fewer barriers.  Thread t loads entries
// t + 512 k (k < 8), so every warp load is one contiguous 256-byte run: index
// bits 9-11 are in registers and bits 0-4 are the lane bits (warp shuffles).
// One shared-memory pass regroups the tile so that each thread holds 8
// entries 32 apart (bits 5-7 in registers), and bit 8 is one shared-memory
// stage.  Sums are order-independent, so every stage is the same add.
template <typename G>
__global__ void __launch_bounds__(kZetaThreads) k_zeta_low12(G* __restrict__ g, size_t n, int32_t* __restrict__ flags) {
  static_assert(kZetaThreads * 8 == (1 << kZetaLowBits), "8 entries per thread");
  __shared__ G t[1 << kZetaLowBits];
  G* tile = g + ((size_t)blockIdx.x << kZetaLowBits);
  if (MPT_BAD(flags, ((size_t)blockIdx.x + 1) << kZetaLowBits <= n)) return;
  const int tid = threadIdx.x, lane = tid & 31;
  G v[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) v[k] = tile[tid + kZetaThreads * k];
#pragma unroll
  for (int j = 0; j < 3; ++j)
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (!(k & (1 << j))) v[k] += v[k | (1 << j)];
#pragma unroll
  for (int j = 0; j < 5; ++j) {
    const bool low = !(lane & (1 << j));  // this lane's entries have bit j clear
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const G o = __shfl_xor_sync(0xFFFFFFFFu, v[k], 1 << j);
      if (low) v[k] += o;
    }
  }
#pragma unroll
  for (int k = 0; k < 8; ++k) t[tid + kZetaThreads * k] = v[k];
  __syncthreads();
  // regroup: thread t takes entries base + 32 k, k < 8 (bits 5-7), with bits
  // 0-4 = t & 31, bit 8 = (t >> 5) & 1 and bits 9-11 = t >> 6
  const int base = lane | (((tid >> 5) & 1) << 8) | ((tid >> 6) << 9);
#pragma unroll
  for (int k = 0; k < 8; ++k) v[k] = t[base + 32 * k];
#pragma unroll
  for (int j = 0; j < 3; ++j)
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (!(k & (1 << j))) v[k] += v[k | (1 << j)];
#pragma unroll
  for (int k = 0; k < 8; ++k) t[base + 32 * k] = v[k];
  __syncthreads();
  // bit 8, then write back
  for (int i = tid; i < (1 << (kZetaLowBits - 1)); i += kZetaThreads) {
    const int e = ((i >> 8) << 9) | (i & 255);  // bit 8 of e clear
    t[e] += t[e | 256];
  }
  __syncthreads();
  for (int i = tid; i < (1 << kZetaLowBits); i += kZetaThreads) tile[i] = t[i];
}

// Superset sums over index bits [lo, lo + tb), tb <= 8: each block owns
// 4096 >> tb adjacent columns (bits below lo, lo >= 12) and all 2^tb values
// of those bits, for one value of the bits above -- 4096 entries, rows of
// contiguous columns.
constexpr int kZetaCols = 16;
constexpr int kZetaHighBits = 8;
constexpr int kZetaBlockEntries = 1 << kZetaLowBits;

template <typename G>
__global__ void __launch_bounds__(kZetaThreads) k_zeta_high(G* __restrict__ g, int lo, int tb, size_t n,
                                                            int32_t* __restrict__ flags) {
  __shared__ G t[kZetaBlockEntries];
  const int cshift = kZetaLowBits - tb;  // log2 of the columns per block
  const int cols = 1 << cshift;
  const size_t col_groups = ((size_t)1 << lo) >> cshift;
  const size_t cg = blockIdx.x % col_groups;
  const size_t top = blockIdx.x / col_groups;
  G* base = g + (top << (lo + tb)) + (cg << cshift);
  // the block's last entry: row 2^tb - 1, its last column
  if (MPT_BAD(flags, (top << (lo + tb)) + ((((size_t)1 << tb) - 1) << lo) + ((cg + 1) << cshift) <= n)) return;
  for (int e = threadIdx.x; e < kZetaBlockEntries; e += blockDim.x) {
    const int r = e >> cshift, c = e & (cols - 1);
    t[e] = base[((size_t)r << lo) + c];
  }
  constexpr int kHalf = kZetaBlockEntries / 2;
  for (int j = 0; j < tb; ++j) {
    __syncthreads();
    const int lowmask = (1 << j) - 1;
    for (int p = threadIdx.x; p < kHalf; p += blockDim.x) {
      const int c = p & (cols - 1), q = p >> cshift;
      const int r = ((q >> j) << (j + 1)) | (q & lowmask);  // bit j of r is 0
      t[(r << cshift) + c] += t[((r | (1 << j)) << cshift) + c];
    }
  }
  __syncthreads();
  for (int e = threadIdx.x; e < kZetaBlockEntries; e += blockDim.x) {
    const int r = e >> cshift, c = e & (cols - 1);
    base[((size_t)r << lo) + c] = t[e];
  }
}

// k_zeta_high for tb = 8 with fewer barriers: thread t owns column t & 15
// and holds 8 rows ((t >> 4) * 8 + i: row bits 0-2 in registers, row bit 3 by
// a warp shuffle); one shared-memory pass regroups so that each thread holds
// rows 16 apart (row bits 4-6 in registers), and row bit 7 is one
// shared-memory stage.
template <typename G>
__global__ void __launch_bounds__(kZetaThreads) k_zeta_high8(G* __restrict__ g, int lo, size_t n,
                                                             int32_t* __restrict__ flags) {
  static_assert(kZetaThreads * 8 == (1 << kZetaHighBits) * kZetaCols, "8 entries per thread");
  __shared__ G t[(1 << kZetaHighBits) * kZetaCols];
  const size_t col_groups = ((size_t)1 << lo) / kZetaCols;
  const size_t cg = blockIdx.x % col_groups;
  const size_t top = blockIdx.x / col_groups;
  G* base = g + (top << (lo + kZetaHighBits)) + cg * kZetaCols;
  if (MPT_BAD(flags, (top << (lo + kZetaHighBits)) + ((((size_t)1 << kZetaHighBits) - 1) << lo) +
                         (cg + 1) * kZetaCols <= n))
    return;
  const int tid = threadIdx.x, c = tid & (kZetaCols - 1), rg = tid >> 4;
  G v[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = base[((size_t)(rg * 8 + i) << lo) + c];
#pragma unroll
  for (int j = 0; j < 3; ++j)
#pragma unroll
    for (int i = 0; i < 8; ++i)
      if (!(i & (1 << j))) v[i] += v[i | (1 << j)];
  {
    const bool low = !(rg & 1);  // row bit 3 clear; the partner row group is lane ^ 16
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const G o = __shfl_xor_sync(0xFFFFFFFFu, v[i], 16);
      if (low) v[i] += o;
    }
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) t[(rg * 8 + i) * kZetaCols + c] = v[i];
  __syncthreads();
  // regroup: rows (rg & 15) | (k << 4) | ((rg >> 4) << 7), k < 8 (row bits 4-6)
  const int r0 = (rg & 15) | ((rg >> 4) << 7);
#pragma unroll
  for (int k = 0; k < 8; ++k) v[k] = t[(r0 | (k << 4)) * kZetaCols + c];
#pragma unroll
  for (int j = 0; j < 3; ++j)
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (!(k & (1 << j))) v[k] += v[k | (1 << j)];
#pragma unroll
  for (int k = 0; k < 8; ++k) t[(r0 | (k << 4)) * kZetaCols + c] = v[k];
  __syncthreads();
  // row bit 7: rows r < 128 take row r + 128
  constexpr int kHalf = (1 << (kZetaHighBits - 1)) * kZetaCols;
  for (int i = tid; i < kHalf; i += kZetaThreads) t[i] += t[i + kHalf];
  __syncthreads();
  for (int e = tid; e < (1 << kZetaHighBits) * kZetaCols; e += kZetaThreads) {
    const int r = e / kZetaCols, cc = e % kZetaCols;
    base[((size_t)r << lo) + cc] = t[e];
  }
}

}  // namespace

cudaError_t launch_scatter(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches) {
  int64_t blocks = (s.n + kScatterThreads - 1) / kScatterThreads;
  const int64_t cap = sm_count() * 16;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  void* g = g_table(s, ws);
  if (s.lean)
    k_scatter<<<(unsigned)blocks, kScatterThreads, 0, stream>>>(
        ws.weights, ws.bits, s.n, s.m, s.words, static_cast<unsigned int*>(g), s.blocked ? ws.priv : nullptr,
        ws.used_N, ws.used_x, ws.counters, s.slots, s.blocked, s.L, s.b);
  else
    k_scatter<<<(unsigned)blocks, kScatterThreads, 0, stream>>>(
        ws.weights, ws.bits, s.n, s.m, s.words, static_cast<unsigned long long*>(g), s.blocked ? ws.priv : nullptr,
        ws.used_N, ws.used_x, ws.counters, s.slots, s.blocked, s.L, s.b);
  ++*launches;
  return cudaGetLastError();
}

template <typename G>
static cudaError_t zeta(const Shape& s, G* g, int32_t* flags, cudaStream_t stream, int* launches) {
  const int tb = s.m < kZetaLowBits ? s.m : kZetaLowBits;
  const size_t low_blocks = (size_t)1 << (s.m - tb);
  const size_t n = (size_t)1 << s.m;
  if (tb == kZetaLowBits)
    k_zeta_low12<<<(unsigned)low_blocks, kZetaThreads, 0, stream>>>(g, n, flags);
  else
    k_zeta_low<<<(unsigned)low_blocks, kZetaThreads, 0, stream>>>(g, tb, n, flags);
  ++*launches;
  cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  for (int lo = tb; lo < s.m; lo += kZetaHighBits) {
    const int hb = (s.m - lo) < kZetaHighBits ? (s.m - lo) : kZetaHighBits;
    const size_t blocks = ((size_t)1 << s.m) / (hb == kZetaHighBits ? ((size_t)1 << hb) * kZetaCols
                                                                      : (size_t)kZetaBlockEntries);
    if (hb == kZetaHighBits)
      k_zeta_high8<<<(unsigned)blocks, kZetaThreads, 0, stream>>>(g, lo, n, flags);
    else
      k_zeta_high<<<(unsigned)blocks, kZetaThreads, 0, stream>>>(g, lo, hb, n, flags);
    ++*launches;
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
  }
  return cudaSuccess;
}

cudaError_t launch_zeta(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches) {
  if (s.lean) return zeta(s, static_cast<unsigned int*>(g_table(s, ws)), ws.counters + 1, stream, launches);
  return zeta(s, static_cast<unsigned long long*>(g_table(s, ws)), ws.counters + 1, stream, launches);
}

}  // namespace mpt
