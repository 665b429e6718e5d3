// K4: hierarchy walk -> layout, and the trie-cost check (Sec. 2, eq. 1).
//
// Layout (Thm 1 proof, "<=" direction): the hierarchy has root {0..m-1};
// node S with |S| >= 2 has children A = split[S] (left) and S \ A (right).
// At node B the chunks of I(B) \ I(parent(B)) are emitted, in increasing chunk
// id, with I(parent(root)) empty.  A chunk x is therefore emitted for request
// i at the highest node B on i's root-to-leaf path with B inside N_x (the
// request set of x), and request i's permutation is R_i sorted by
// (depth of that node, chunk id).  The left-to-right leaf order is the trie
// DFS order that Thm 7 (Sec. 8) serves requests in.  After a blocked solve
// split is read at the rotated position of each node and OPT = F(full) =
// F'(full) + sum_i pi_i + u from Gp = F' << b (uint32, or uint64 on the wide
// path) and the offsets pi, u (k_scatter_zeta.cu); after a general one both
// are in natural order.
//
// Trie cost: a string's node at depth p is new exactly when no earlier
// string shares its first p+1 symbols, so the trie weight is
//     sum_i sum over positions p >= max_{j<i} lcp(i, j) of w(seq_i[p]).
#include "mpt_internal.cuh"

namespace mpt {
namespace {

constexpr int kWalkThreads = 256;
constexpr int kMaxM = 32;

__global__ void __launch_bounds__(kWalkThreads)
k_walk(int m, const uint32_t* __restrict__ split, const int64_t* __restrict__ F, const int32_t* __restrict__ F32,
       const uint32_t* __restrict__ Gp, const unsigned long long* __restrict__ Gp64,
       const unsigned long long* __restrict__ priv, int L, int b, const uint32_t* __restrict__ used_N,
       const int32_t* __restrict__ used_x, int32_t* __restrict__ counters, int64_t slots,
       unsigned long long* __restrict__ keys, int64_t* __restrict__ perm_offsets, int64_t* __restrict__ perm_chunks,
       int32_t* __restrict__ dfs, int64_t* __restrict__ opt) {
  __shared__ uint32_t anc[kMaxM][kMaxM];  // anc[i][d]: the depth-d node on request i's path
  __shared__ int leaf_depth[kMaxM];
  __shared__ int cnt[kMaxM];
  __shared__ int fill[kMaxM];
  __shared__ long long offs[kMaxM + 1];
  __shared__ int bad;

  const int tid = threadIdx.x;
  if (tid < kMaxM) {
    cnt[tid] = 0;
    fill[tid] = 0;
    leaf_depth[tid] = 0;
  }
  if (tid == 0) {
    bad = 0;
    const uint32_t full = (m >= 32) ? 0xFFFFFFFFu : ((1u << m) - 1u);
    uint32_t stk[2 * kMaxM];
    int stk_d[2 * kMaxM];
    int sp = 0, nleaf = 0;
    stk[sp] = full;
    stk_d[sp] = 0;
    ++sp;
    while (sp > 0 && !bad) {
      --sp;
      const uint32_t S = stk[sp];
      const int d = stk_d[sp];
      for (uint32_t r = S; r; r &= r - 1) anc[__ffs(r) - 1][d] = S;
      if ((S & (S - 1)) == 0) {
        const int i = __ffs(S) - 1;
        leaf_depth[i] = d;
        dfs[nleaf++] = i;
        continue;
      }
      // blocked path: split and F (as F << b in Gp) in rotated order
      const uint32_t A = (Gp || Gp64) ? split[rot_index(S, L, b)] : split[S];
      if (A == 0 || (A & ~S) != 0 || A == S || sp + 2 > 2 * kMaxM) {
        bad = 1;
        break;
      }
      stk[sp] = S ^ A;  // right child, visited after the left subtree
      stk_d[sp] = d + 1;
      ++sp;
      stk[sp] = A;
      stk_d[sp] = d + 1;
      ++sp;
    }
    if (bad) atomicOr(&counters[1], kErrBadSplit);
    int64_t pi_all = 0;
    if (priv) {
      for (int i = 0; i < m; ++i) pi_all += (int64_t)priv[i];
      pi_all += (int64_t)priv[kUniversalSlot];
    }
    *opt = Gp64 ? (int64_t)(Gp64[rot_index(full, L, b)] >> b) + pi_all
           : Gp ? (int64_t)(Gp[rot_index(full, L, b)] >> b) + pi_all
                : (F ? F[full] : (int64_t)F32[full]);
  }
  __syncthreads();
  if (bad) return;

  int used = counters[0];
  if (used > slots) used = (int)slots;
  for (int t = tid; t < used; t += kWalkThreads)
    for (uint32_t r = used_N[t]; r; r &= r - 1) atomicAdd(&cnt[__ffs(r) - 1], 1);
  __syncthreads();
  if (tid == 0) {
    long long acc = 0;
    for (int i = 0; i < m; ++i) {
      offs[i] = acc;
      perm_offsets[i] = acc;
      acc += cnt[i];
    }
    offs[m] = acc;
    perm_offsets[m] = acc;
    if (acc != slots) atomicOr(&counters[1], kErrLayoutCount);
  }
  __syncthreads();

  for (int t = tid; t < used; t += kWalkThreads) {
    const uint32_t N = used_N[t];
    const unsigned long long x = (unsigned long long)(uint32_t)used_x[t];
    for (uint32_t r = N; r; r &= r - 1) {
      const int i = __ffs(r) - 1;
      int d = 0;
      while (d < leaf_depth[i] && (anc[i][d] & ~N) != 0) ++d;
      const int slot = atomicAdd(&fill[i], 1);
      if (offs[i] + slot < slots) keys[offs[i] + slot] = ((unsigned long long)d << 32) | x;
    }
  }
  __syncthreads();

  const int lane = tid & 31, warp = tid >> 5;
  for (int i = warp; i < m; i += kWalkThreads / 32) {
    const long long base = offs[i];
    const int len = cnt[i];
    for (int j = lane; j < len; j += 32) {
      const unsigned long long kj = keys[base + j];
      int rank = 0;
      for (int t = 0; t < len; ++t) rank += keys[base + t] < kj;
      perm_chunks[base + rank] = (int64_t)(kj & 0xFFFFFFFFull);
    }
  }
}

__global__ void __launch_bounds__(kWalkThreads)
k_trie_cost(int m, const int64_t* __restrict__ w, const int64_t* __restrict__ offs, const int64_t* __restrict__ seq,
            int64_t* __restrict__ cost) {
  __shared__ int maxlcp[kMaxM];
  __shared__ unsigned long long total;
  const int tid = threadIdx.x;
  if (tid < kMaxM) maxlcp[tid] = 0;
  if (tid == 0) total = 0;
  __syncthreads();
  for (int p = tid; p < m * m; p += kWalkThreads) {
    const int i = p / m, j = p % m;
    if (j >= i) continue;
    const int64_t li = offs[i + 1] - offs[i], lj = offs[j + 1] - offs[j];
    const int64_t lim = li < lj ? li : lj;
    int64_t l = 0;
    while (l < lim && seq[offs[i] + l] == seq[offs[j] + l]) ++l;
    atomicMax(&maxlcp[i], (int)l);
  }
  __syncthreads();
  for (int i = tid; i < m; i += kWalkThreads) {
    unsigned long long s = 0;
    for (int64_t p = offs[i] + maxlcp[i]; p < offs[i + 1]; ++p) s += (unsigned long long)w[seq[p]];
    atomicAdd(&total, s);
  }
  __syncthreads();
  if (tid == 0) *cost = (int64_t)total;
}

}  // namespace

cudaError_t launch_walk(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches) {
  k_walk<<<1, kWalkThreads, 0, stream>>>(s.m, s.blocked ? ws.split_rot : ws.split, s.lean ? nullptr : ws.F,
                                         s.lean ? ws.fw : nullptr, s.blocked && !s.wide ? ws.Gp : nullptr,
                                         s.blocked && s.wide ? ws.Gp64 : nullptr, s.blocked ? ws.priv : nullptr,
                                         s.L, s.b, ws.used_N,
                                         ws.used_x, ws.counters, s.slots, ws.keys,
                                         ws.perm_offsets, ws.perm_chunks, ws.dfs, ws.opt);
  ++*launches;
  return cudaGetLastError();
}

cudaError_t launch_trie_cost(int m, const int64_t* d_weights, const int64_t* d_offsets, const int64_t* d_chunks,
                             int64_t* d_cost, cudaStream_t stream) {
  k_trie_cost<<<1, kWalkThreads, 0, stream>>>(m, d_weights, d_offsets, d_chunks, d_cost);
  return cudaGetLastError();
}

}  // namespace mpt
