// Batched exact solve of many small instances (m <= 15 requests each), one
// block per instance with its tables in shared memory: the row-blocked
// kernel for packed keys (m >= 6), the per-subset kernel otherwise.
//
// This is the paper's own use of the exact recurrence (Sec. 6.2: 72 synthetic
// groups of 10-15 requests; Sec. 7: real request groups of at most 13): many
// independent groups, each small enough that its 2^m tables fit on chip.
// Per block, in order:
//   1. gather the instance's (chunk, request) occurrences into a hash table
//      in shared memory, so that each distinct chunk x gets its request set
//      N_x (S_x of Sec. 3) by OR-ing its requests;
//   2. g(T) = sum of w(x) over N_x = T, then superset sums: wI(S) = w(I(S)),
//      in the F table itself: entry S holds w(I(S)) until the recurrence
//      finishes S and writes F(S) over it (only S's finisher reads w(I(S)),
//      and F is read only at finished subsets of lower layers);
//   3. the Sec. 3.1 recurrence layer by layer, F(S) = min over splits of
//      F(A) + F(S \ A) - wI(S), the split named by its part A holding the
//      lowest request of S and the smallest such A kept on ties;
//   4. the hierarchy walk of the Thm 1 proof: request i's chunks ordered by
//      (depth of the highest node on its path inside N_x, chunk id), and the
//      left-to-right leaf order (Thm 7).
// Offsets: a chunk that one request alone holds, or that all m >= 2 hold, is
// one cluster in every hierarchy (Thm 1), so for instances whose
// sum_i w(R_i) would not fit the packed keys (flag kFlagOffsets) step 2 adds
// it to a per-request sum pi_i or a universal sum u instead of to g, step 3
// runs on F'(S) = F(S) - sum_{i in S} pi_i - u, and the outputs add those
// back (the same reduction as the single-instance scatter,
// k_scatter_zeta.cu).  Lighter instances keep the plain form (F' = F).
// Values are kept in 32 bits: the host accepts an instance only when its
// shared weight W = sum_i w(R_i) - sum_i pi_i - m u is below 2^31, so every
// F' and every split sum fits.  When also W < 2^(32-m) (the common case),
// the F table holds F' << m and the
// key of split A is F[A] + F[S \ A] + A = ((F(A) + F(S \ A)) << m) + A: one
// 32-bit minimum picks the least value and, among equal values, the least A.
// Otherwise keys are (value << 16 | A) in 64 bits.
// The host launches one grid per instance size m (blocks indexed through a
// list of instances), so that shared memory is sized for that m.
#include "mpt_internal.cuh"

namespace mpt {
namespace {

constexpr int kBatchThreads = 256;
constexpr int kBatchOffsets = 17;  // pi_i in slots 0..m-1 (m <= 15), u in slot kBatchUniv
constexpr int kBatchUniv = 16;

// Step 2's scatter: chunk u of the instance goes to pi_i (N_x = {i}), to u
// (N_x = all m >= 2 requests) or to g(N_x), the last through g_at(N_x); with
// off null, every chunk goes to g.
template <int TPI, typename GAt>
__device__ void batch_scatter(int m, int nd, const int64_t* __restrict__ weights, const int32_t* cx,
                              const uint32_t* cN, unsigned long long* off, GAt g_at) {
  for (int u = threadIdx.x; u < nd; u += TPI) {
    const uint32_t Nx = cN[u];
    const unsigned long long wx = (unsigned long long)weights[cx[u]];
    if (off && (Nx & (Nx - 1)) == 0)
      atomicAdd(&off[__ffs(Nx) - 1], wx);
    else if (off && __popc(Nx) == m)  // all m requests (written this way, ptxas keeps k_batch_rows spill-free)
      atomicAdd(&off[kBatchUniv], wx);
    else
      atomicAdd(g_at(Nx), (uint32_t)wx);
  }
}

// What step 3 left out of F(S): sum_{i in S} pi_i + u for S non-empty.  A
// thread writes the entries S = t, t + TPI, t + 2 TPI, ..., so the requests
// below TPI are its own (summed once, lo) and only the others are summed per
// entry.
__device__ __forceinline__ int64_t batch_pi(uint32_t S, const unsigned long long* off) {
  int64_t v = 0;
  for (uint32_t r = S; r; r &= r - 1) v += (int64_t)off[__ffs(r) - 1];
  return v;
}
template <int TPI>
__device__ __forceinline__ int64_t batch_offset(uint32_t S, int64_t lo, const long long* hi) {
  return S == 0 ? 0 : lo + hi[S / TPI];
}


// Step 1: the instance's distinct chunks cx[0..nd) (in no particular order)
// with their request sets cN -- N_x = S_x of Sec. 3 -- through a hash table
// in shared memory: tkey[0..2*occ_cap) (chunk id or -1) and tmask (request
// bits), open addressing with linear probing.  The table has at least twice
// as many slots as occurrences, so every insertion ends within `size` probes.
template <int TPI>
__device__ int batch_gather(int m, int64_t r0, int64_t o0, int occ, int occ_cap, const int64_t* __restrict__ req_off,
                            const int64_t* __restrict__ chunks, int32_t* tkey, uint32_t* tmask, int32_t* cx,
                            uint32_t* cN, int* roff, int* ndistinct_s, int32_t* bflags) {
  int& ndistinct = *ndistinct_s;
  const int t = threadIdx.x;
  const int size = 2 * occ_cap;  // a power of two
  const int lg = 31 - __clz(size);
  if (t == 0) ndistinct = 0;
  if (t <= m) roff[t] = (int)(req_off[r0 + t] - o0);
  for (int h = t; h < size; h += TPI) {
    tkey[h] = -1;
    tmask[h] = 0;
  }
  __syncthreads();
  for (int j = t; j < occ; j += TPI) {
    int i = 0;
    while (roff[i + 1] <= j) ++i;  // the request whose slot range holds j
    const int32_t x = (int32_t)chunks[o0 + j];
    uint32_t h = lg > 0 ? ((uint32_t)x * 2654435761u) >> (32 - lg) : 0u;
    for (int probe = 0; probe < size; ++probe) {
      const int32_t old = atomicCAS(&tkey[h], -1, x);
      if (old == -1 || old == x) {
        atomicOr(&tmask[h], 1u << i);
        break;
      }
      h = (h + 1u) & (uint32_t)(size - 1);
    }
  }
  __syncthreads();
  for (int h = t; h < size; h += TPI) {
    const int32_t x = tkey[h];
    if (x >= 0) {
      const int u = atomicAdd(&ndistinct, 1);
      if (MPT_BAD(bflags, u < occ_cap)) continue;
      cx[u] = x;
      cN[u] = tmask[h];
    }
  }
  __syncthreads();
  return ndistinct;
}

// Step 4: the hierarchy walk of the Thm 1 proof from the split table
// (split(S) for S = 0 .. 2^m - 1; shared or global), the permutations and the
// left-to-right leaf order.  Every thread of the block calls it after the
// split table is complete and visible.
// roff: the request offsets staged by batch_gather (shared memory).
template <int TPI, typename SplitT>
__device__ void batch_walk(int inst, int m, int64_t r0, int64_t o0, const int* roff, const SplitT* split,
                           unsigned long long* keys, const int32_t* cx, const uint32_t* cN, int nd,
                           int64_t* __restrict__ perm_out, int32_t* __restrict__ dfs_out,
                           int32_t* __restrict__ status) {
  __shared__ uint32_t anc[16][16];
  __shared__ int leaf_depth[16], fill[16], dfs_s[16];
  __shared__ int bad;
  const int t = threadIdx.x;
  const int N = 1 << m;
  if (t < 16) {
    fill[t] = 0;
    leaf_depth[t] = 0;
  }
  if (t == 0) {
    bad = 0;
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
      const uint32_t A = (uint32_t)split[S];
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
  for (int u = t; u < nd; u += TPI) {
    const uint32_t Nx = cN[u];
    for (uint32_t rr = Nx; rr; rr &= rr - 1) {
      const int i = __ffs(rr) - 1;
      int d = 0;
      while (d < leaf_depth[i] && (anc[i][d] & ~Nx) != 0) ++d;
      const int slot = atomicAdd(&fill[i], 1);
      keys[roff[i] + slot] = ((unsigned long long)d << 32) | (unsigned long long)(uint32_t)cx[u];
    }
  }
  __syncthreads();
  const int lane = t & 31, warp = t >> 5;
  for (int i = warp; i < m; i += TPI / 32) {
    const int base = roff[i];
    const int len = roff[i + 1] - roff[i];
    for (int j = lane; j < len; j += 32) {
      const unsigned long long kj = keys[base + j];
      int rank = 0;
      for (int q = 0; q < len; ++q) rank += keys[base + q] < kj;
      perm_out[o0 + base + rank] = (int64_t)(kj & 0xFFFFFFFFull);
    }
  }
  if (t == 0) status[inst] = 0;
}

__global__ void __launch_bounds__(kBatchThreads)
k_batch_solve(const int64_t* __restrict__ weights, const int64_t* __restrict__ inst_req,
              const int64_t* __restrict__ req_off, const int64_t* __restrict__ chunks,
              const int64_t* __restrict__ tab_off, const int32_t* __restrict__ inst_list,
              const uint8_t* __restrict__ flags, int occ_cap, int max_m, int64_t* __restrict__ opt_out,
              int64_t* __restrict__ F_out, uint32_t* __restrict__ split_out, int64_t* __restrict__ perm_out,
              int32_t* __restrict__ dfs_out, int32_t* __restrict__ status) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int inst = inst_list[blockIdx.x];
  const bool packed = (flags[inst] & kFlagPacked) != 0;
  const bool use_off = (flags[inst] & kFlagOffsets) != 0;
  const int64_t r0 = inst_req[inst], r1 = inst_req[inst + 1];
  const int m = (int)(r1 - r0);
  const int64_t o0 = req_off[r0], o1 = req_off[r1];
  const int occ = (int)(o1 - o0);
  const int N = 1 << m;

  // shared layout (sized for max_m and occ_cap by the host)
  unsigned long long* keys = reinterpret_cast<unsigned long long*>(smem_raw);  // [occ_cap] sort keys, later walk keys
  uint32_t* F = reinterpret_cast<uint32_t*>(keys + occ_cap);                   // [2^max_m] w(I(S)), then F(S)
  uint32_t* wI = F;
  uint16_t* split = reinterpret_cast<uint16_t*>(F + (1 << max_m));             // [2^max_m]
  int32_t* cx = reinterpret_cast<int32_t*>(split + (1 << max_m));              // [occ_cap] distinct chunk ids
  uint32_t* cN = reinterpret_cast<uint32_t*>(cx + occ_cap);                    // [occ_cap] their request sets
  uint32_t* tmask = cN + occ_cap;                                                // [2 * occ_cap] hash-table masks
  __shared__ int ndistinct;
  __shared__ int roff[17];  // request offsets relative to o0 (m + 1 <= 17)
  __shared__ unsigned long long off[kBatchOffsets];
  __shared__ int32_t bflags;  // bounds-checked build: failed checks of this block
  const int t = threadIdx.x;
  // the shared arrays were sized for max_m and occ_cap (the same decision in
  // every thread)
  if (MPT_BAD(&bflags, m >= 1 && m <= max_m && occ <= occ_cap)) {
    if (t == 0) status[inst] = kErrBounds;
    return;
  }
  if (t == 0) bflags = 0;
  const int nd = batch_gather<kBatchThreads>(m, r0, o0, occ, occ_cap, req_off, chunks,
                                             reinterpret_cast<int32_t*>(keys), tmask, cx, cN, roff, &ndistinct,
                                             &bflags);
  for (int S = t; S < N; S += kBatchThreads) wI[S] = 0;
  if (t < kBatchOffsets) off[t] = 0;
  __syncthreads();

  // 2. g(T) and the offsets, then superset sums over the m request bits
  batch_scatter<kBatchThreads>(m, nd, weights, cx, cN, use_off ? off : nullptr,
                               [&](uint32_t Nx) { return &wI[Nx]; });
  __syncthreads();
  for (int j = 0; j < m; ++j) {
    for (int p = t; p < (N >> 1); p += kBatchThreads) {
      const int S = ((p >> j) << (j + 1)) | (p & ((1 << j) - 1));
      wI[S] += wI[S | (1 << j)];
    }
    __syncthreads();
  }

  // 3. the recurrence, one popcount layer at a time
  const int vshift = packed ? m : 0;  // F holds F << vshift
  for (int S = t; S < N; S += kBatchThreads) {
    if ((S & (S - 1)) == 0) {
      F[S] = S ? wI[S] << vshift : 0u;
      split[S] = 0;
    }
  }
  __syncthreads();
  for (int k = 2; packed && k <= m; ++k) {
    const int count = (int)c_binom.v[m][k];
    // lanes per subset: enough to keep the block busy, at most 32; lanes
    // split the parts on the LOWEST bits of S \ lowbit(S), so the lanes of a
    // subset read F at different banks whenever those requests are low
    int g = 0;
    while ((count << (g + 1)) <= kBatchThreads && g < 5 && g < k - 1) ++g;
    const int G = 1 << g;
    const int per_pass = kBatchThreads >> g;
    for (int base = 0; base < count; base += per_pass) {
      const int idx = base + (t >> g);
      const uint32_t r = (uint32_t)t & (uint32_t)(G - 1);
      uint32_t best = 0xFFFFFFFFu;
      uint32_t S = 0;
      if (idx < count) {
        S = colex_unrank((unsigned long long)idx, k, m);
        const uint32_t low = S & (~S + 1u);
        const uint32_t rest = S ^ low;
        uint32_t lo = 0, rr = rest;
        for (int q = 0; q < g; ++q) {
          const uint32_t lb = rr & (~rr + 1u);
          lo |= lb;
          rr ^= lb;
        }
        const uint32_t freem = rest ^ lo;
        const uint32_t fixed = deposit_bits(r, lo);
        const uint32_t lowfixed = low | fixed;
        const bool last_lane = fixed == lo;  // only this lane meets part == rest (A = S)
        uint32_t sub = 0;
        do {
          const uint32_t A = lowfixed | sub;
          if (!(last_lane && sub == freem)) best = min(best, F[A] + F[S ^ A] + A);
          sub = (sub - freem) & freem;
        } while (sub != 0);
      }
      for (int off = G >> 1; off > 0; off >>= 1) best = min(best, __shfl_xor_sync(0xFFFFFFFFu, best, off));
      if (idx < count && r == 0) {
        F[S] = ((best >> m) - wI[S]) << m;
        split[S] = (uint16_t)(best & (uint32_t)(N - 1));
        (void)MPT_BAD(&bflags, valid_split(S, best & (uint32_t)(N - 1)));
      }
    }
    __syncthreads();
  }
  for (int k = 2; !packed && k <= m; ++k) {
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
        (void)MPT_BAD(&bflags, valid_split(S, (uint32_t)(best & 0xFFFFu)));
      }
    }
    __syncthreads();
  }

  // outputs: tables and OPT
  const int64_t tb = tab_off[inst];
  if (use_off) {
    __shared__ long long hi_off[(1 << 15) / kBatchThreads];
    for (int i = t; i < (N + kBatchThreads - 1) / kBatchThreads; i += kBatchThreads)
      hi_off[i] = batch_pi((uint32_t)i * kBatchThreads, off) + (long long)off[kBatchUniv];
    __syncthreads();
    const int64_t lo = batch_pi((uint32_t)t & (kBatchThreads - 1), off);
    for (int S = t; S < N; S += kBatchThreads) {
      F_out[tb + S] = (int64_t)(F[S] >> vshift) + batch_offset<kBatchThreads>((uint32_t)S, lo, hi_off);
      split_out[tb + S] = split[S];
    }
    if (t == 0)
      opt_out[inst] = (int64_t)(F[N - 1] >> vshift) + batch_pi((uint32_t)N - 1u, off) + (int64_t)off[kBatchUniv];
  } else {
    for (int S = t; S < N; S += kBatchThreads) {
      F_out[tb + S] = (int64_t)(F[S] >> vshift);
      split_out[tb + S] = split[S];
    }
    if (t == 0) opt_out[inst] = (int64_t)(F[N - 1] >> vshift);
  }

  // 4. hierarchy walk
  __syncthreads();
  batch_walk<kBatchThreads>(inst, m, r0, o0, roff, split, keys, cx, cN, nd, perm_out, dfs_out, status);
  if (kBoundsChecked) {
    __syncthreads();
    if (t == 0 && bflags) status[inst] = bflags;
  }
}

// ---------------------------------------------------------------------------
// Row-blocked recurrence for instances with m >= 6 and packed keys.
//
// The 2^m subsets U = (s1, s2) are 2^(m-5) rows s1 of 32 entries s2, stored
// at row_pos(s1) * 36 + s2 (rows padded to 36 words and XOR-placed so that
// the 16-byte chunks of different rows fall in different bank groups).  The
// keys are
//   Gp(X) = (F(X) << m) + X,   Gc(X) = F(X) << m = Gp(X) - X,
// so Gp(A) + Gc(B) = ((F(A) + F(B)) << m) + A: an unsigned min over splits
// picks the least value and, among equal values, the least A.  Only Gp is
// stored; a row is turned into its Gc form when it is loaded.  Before U is
// finished, Gp(U) holds w(I(U)) (superset sums in place).
// A split of U names the part A holding lowbit(U):
//   * s2 != 0: A = (a1, a2) with a2 holding lowbit(s2), any a1 within s1;
//     - a1 not in {0, s1}: rows a1 and s1 ^ a1 were finished at an earlier
//       level of |s1| -- a register convolution of two rows restricted to
//       a2 holding lowbit(s2) (121 add-min pairs);
//     - a1 = 0 (B in this row) and a1 = s1 (A in this row, a2 != s2): the
//       in-row recurrence, in increasing s2, in registers;
//   * s2 = 0: A = (a1, 0) with a1 holding lowbit(s1), a1 != s1 -- the
//     entry-0 column of the same row pairs.
// Levels go by |s1|; within a level, phase A (row pairs, several lanes per
// row) then phase B (one thread per row finishes it).
// ---------------------------------------------------------------------------
constexpr int kBRow = 32;
constexpr int kBRowStride = 36;
constexpr int kBMaxLevelRows = 462;  // C(11, 5): the most rows of one level (m = 16)
constexpr int kBMaxRowsM = 16;
constexpr int kBGlobalRowsM = 16;    // from here the rows live in a global scratch slot per block
constexpr int kBGlobalSplitM = 14;   // from here the split table goes straight to global memory
constexpr int kBkStride = kBRow + 1; // phase A minima: 33 words a row, so rows read by one warp use different banks

// rows of the largest level C(nb, nb / 2), rounded up to even so that the
// 64-bit keys after the minima stay 8-byte aligned
__host__ __device__ constexpr int batch_level_rows(int nb) {
  int c = 1;
  for (int i = 0; i < nb / 2; ++i) c = c * (nb - i) / (i + 1);
  return (c + 1) & ~1;
}
static_assert(batch_level_rows(kBMaxRowsM - 5) == kBMaxLevelRows, "the most rows of one level (m = 16)");

// threads per block of the row-blocked kernel for m requests: enough lanes for
// the busiest level (rows x lanes per row) -- 30 up to m = 11, 84 at m = 12,
// 224 at m = 13; from m = 14 the 256 threads take a level's lanes in passes
constexpr int batch_rows_threads(int m) { return m <= 11 ? 64 : (m == 12 ? 128 : 256); }

// lanes per row in phase A at row level p1: enough that each lane runs at
// most 8 row pairs, but no more than a warp (the lanes of a row reduce with
// shuffles)
__host__ __device__ constexpr int batch_rows_g(int p1) { return p1 <= 3 ? 0 : (p1 - 3 < 5 ? p1 - 3 : 5); }

// lanes the busiest level needs: rows C(nb, p1) times 2^g lanes per row in
// phase A, C(nb, p1) threads in phase B
constexpr int batch_rows_lanes(int nb) {
  int most = 0;
  for (int p1 = 1; p1 <= nb; ++p1) {
    int c = 1;
    for (int i = 0; i < p1; ++i) c = c * (nb - i) / (i + 1);
    const int lanes = c * (1 << batch_rows_g(p1));
    most = lanes > most ? lanes : most;
  }
  return most;
}
// Up to m = 13 every level's lanes fit the block in one pass, beyond it
// phase A runs in passes; phase B has one thread per row in one pass up to
// m = 15 and runs in passes at m = 16.
constexpr bool batch_rows_fit() {
  for (int m = 6; m <= 13; ++m)
    if (batch_rows_lanes(m - 5) > batch_rows_threads(m)) return false;
  for (int m = 6; m < kBGlobalRowsM; ++m)
    if (batch_level_rows(m - 5) > batch_rows_threads(m)) return false;
  return true;
}
static_assert(batch_rows_fit(), "every level of the row-blocked kernel fits its block");

// entries of the per-block offset table (one per TPI subsets) of each
// variant: m <= 12 on 64 and 128 threads, m <= 15 on 256, m = 16 with the
// rows in global memory
__host__ __device__ constexpr int batch_rows_hi_entries(int tpi, bool grows) {
  return grows ? (1 << kBGlobalRowsM) / 256 : (tpi == 256 ? (1 << (kBGlobalRowsM - 1)) / 256 : 32);
}
constexpr bool batch_rows_hi_fit() {
  for (int m = 6; m <= kBMaxRowsM; ++m)
    if ((1 << m) / batch_rows_threads(m) > batch_rows_hi_entries(batch_rows_threads(m), m >= kBGlobalRowsM))
      return false;
  return true;
}
static_assert(batch_rows_hi_fit(), "the offset table covers every size of each block width");

__device__ __forceinline__ int brow_pos(uint32_t r) { return (int)(r ^ (((r >> 3) ^ (r >> 6)) & 7u)); }
__device__ __forceinline__ int bidx(uint32_t U) { return brow_pos(U >> 5) * kBRowStride + (int)(U & 31u); }

__device__ __forceinline__ void bload_row(uint32_t (&v)[kBRow], const uint32_t* p) {
  const uint4* q = reinterpret_cast<const uint4*>(p);
#pragma unroll
  for (int c = 0; c < kBRow / 4; ++c) {
    const uint4 t = q[c];
    v[4 * c] = t.x;
    v[4 * c + 1] = t.y;
    v[4 * c + 2] = t.z;
    v[4 * c + 3] = t.w;
  }
}

__device__ __forceinline__ void bstore_row(uint32_t* p, const uint32_t (&v)[kBRow]) {
  uint4* q = reinterpret_cast<uint4*>(p);
#pragma unroll
  for (int c = 0; c < kBRow / 4; ++c) q[c] = make_uint4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
}

// acc[s2] = min over a2 within s2 holding lowbit(s2) of x[a2] + y[s2 ^ a2], s2 = 1..31
__device__ __forceinline__ void bconv_restricted(uint32_t (&acc)[kBRow], const uint32_t (&x)[kBRow],
                                                 const uint32_t (&y)[kBRow]) {
#pragma unroll
  for (int a2 = 1; a2 < kBRow; ++a2) {
#pragma unroll
    for (int s2 = 1; s2 < kBRow; ++s2) {
      if ((a2 & s2) == a2 && (a2 & (s2 & -s2)) != 0) acc[s2] = min(acc[s2], x[a2] + y[s2 ^ a2]);
    }
  }
}

template <int TPI, bool kGRows = false>
__global__ void __launch_bounds__(TPI, TPI >= 256 ? 3 : (TPI == 128 ? 6 : 12))  // 12 warps or more per SM
k_batch_rows(const int64_t* __restrict__ weights, const int64_t* __restrict__ inst_req,
             const int64_t* __restrict__ req_off, const int64_t* __restrict__ chunks,
             const int64_t* __restrict__ tab_off, const int32_t* __restrict__ inst_list,
             const uint8_t* __restrict__ flags, int occ_cap, int mm, int64_t* __restrict__ opt_out,
             int64_t* __restrict__ F_out, uint32_t* __restrict__ split_out, int64_t* __restrict__ perm_out,
             int32_t* __restrict__ dfs_out, int32_t* __restrict__ status, uint32_t* __restrict__ rows_scratch) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int inst = inst_list[blockIdx.x];
  const int64_t r0 = inst_req[inst], r1 = inst_req[inst + 1];
  const int m = (int)(r1 - r0);  // == mm
  const int64_t o0 = req_off[r0], o1 = req_off[r1];
  const int occ = (int)(o1 - o0);
  const int N = 1 << m;
  const int nb = m - 5;
  const int R = 1 << nb;
  const uint32_t mask = (uint32_t)N - 1u;
  const int64_t tb = tab_off[inst];

  // Gp(X) = (F(X) << m) + X only: the complement form Gc(X) = Gp(X) - X is
  // formed from it when a row is loaded
  // (kGRows: the rows, 295 KB at m = 16, live in this block's slot of a
  // global scratch array instead, L1/L2-resident while the block runs)
  const size_t row_words = (size_t)(1 << (mm - 5)) * kBRowStride;
  uint32_t* Gp = kGRows ? rows_scratch + (size_t)blockIdx.x * row_words
                        : reinterpret_cast<uint32_t*>(smem_raw);                 // [R * 36]
  uint32_t* bk = kGRows ? reinterpret_cast<uint32_t*>(smem_raw) : Gp + row_words;  // [level rows * 33] phase A minima
  unsigned long long* keys =
      reinterpret_cast<unsigned long long*>(bk + batch_level_rows(mm - 5) * kBkStride);  // [occ_cap]
  int32_t* cx = reinterpret_cast<int32_t*>(keys + occ_cap);                        // [occ_cap]
  uint32_t* cN = reinterpret_cast<uint32_t*>(cx + occ_cap);                        // [occ_cap]
  uint32_t* tmask = cN + occ_cap;                                                  // [2 * occ_cap] hash-table masks
  uint16_t* split = reinterpret_cast<uint16_t*>(tmask + 2 * occ_cap);              // [2^m] for the walk (m < 14)
  // from m = 14 the split table is written to its output slots directly and
  // the walk reads it there
  const bool gsplit = mm >= kBGlobalSplitM;
  uint32_t* gsp = split_out + tab_off[inst];
  auto put_split = [&](uint32_t U, uint32_t A, int32_t* bf) {
    (void)MPT_BAD(bf, valid_split(U, A));
    if (gsplit)
      gsp[U] = A;
    else
      split[U] = (uint16_t)A;
  };
  __shared__ int ndistinct;
  const int t = threadIdx.x;

  __shared__ int roff[17];  // request offsets relative to o0 (m + 1 <= 17)
  __shared__ unsigned long long off[kBatchOffsets];
  __shared__ int32_t bflags;  // bounds-checked build: failed checks of this block
  // the shared arrays and the rows were sized for mm and occ_cap (the same
  // decision in every thread)
  if (MPT_BAD(&bflags, m == mm && occ <= occ_cap && (!kGRows || rows_scratch))) {
    if (t == 0) status[inst] = kErrBounds;
    return;
  }
  if (t == 0) bflags = 0;
  const int nd = batch_gather<TPI>(m, r0, o0, occ, occ_cap, req_off, chunks, reinterpret_cast<int32_t*>(keys), tmask,
                                   cx, cN, roff, &ndistinct, &bflags);

  // g, the offsets and the superset sums, in the padded row layout: the five
  // in-row bits per row in registers, then one row-pair pass per row bit
  for (int i = t; i < R * kBRowStride; i += TPI) Gp[i] = 0;
  if (t < kBatchOffsets) off[t] = 0;
  __syncthreads();
  const bool use_off = (flags[inst] & kFlagOffsets) != 0;
  batch_scatter<TPI>(m, nd, weights, cx, cN, use_off ? off : nullptr, [&](uint32_t Nx) { return &Gp[bidx(Nx)]; });
  __syncthreads();
  for (int r = t; r < R; r += TPI) {
    uint32_t v[kBRow];
    uint32_t* row = Gp + brow_pos((uint32_t)r) * kBRowStride;
    bload_row(v, row);
#pragma unroll
    for (int j = 0; j < 5; ++j)
#pragma unroll
      for (int x = 0; x < kBRow; ++x)
        if (!(x & (1 << j))) v[x] += v[x | (1 << j)];
    bstore_row(row, v);
  }
  __syncthreads();
  for (int jr = 0; jr < nb; ++jr) {
    for (int p = t; p < (R >> 1); p += TPI) {
      const uint32_t r = (uint32_t)(((p >> jr) << (jr + 1)) | (p & ((1 << jr) - 1)));
      uint32_t v[kBRow], u[kBRow];
      uint32_t* row = Gp + brow_pos(r) * kBRowStride;
      bload_row(v, row);
      bload_row(u, Gp + brow_pos(r | (1u << jr)) * kBRowStride);
#pragma unroll
      for (int x = 0; x < kBRow; ++x) v[x] += u[x];
      bstore_row(row, v);
    }
    __syncthreads();
  }

  // level 0: row 0, the recurrence on the five low requests
  if (t == 0) {
    uint32_t zp[kBRow], zc[kBRow];
#pragma unroll
    for (int s2 = 0; s2 < kBRow; ++s2) {
      const uint32_t wv = Gp[s2];
      uint32_t f, A;
      if (s2 == 0) {
        f = 0;
        A = 0;
      } else if ((s2 & (s2 - 1)) == 0) {
        f = wv;
        A = 0;
      } else {
        uint32_t key = 0xFFFFFFFFu;
#pragma unroll
        for (int a2 = 1; a2 < kBRow; ++a2)
          if ((a2 & s2) == a2 && (a2 & (s2 & -s2)) != 0 && a2 != s2) key = min(key, zp[a2] + zc[s2 ^ a2]);
        f = (key >> m) - wv;
        A = key & mask;
      }
      zp[s2] = (f << m) + (uint32_t)s2;
      zc[s2] = f << m;
      put_split((uint32_t)s2, A, &bflags);
    }
#pragma unroll
    for (int s2 = 0; s2 < kBRow; ++s2) Gp[s2] = zp[s2];
  }
  __syncthreads();

  for (int p1 = 1; p1 <= nb; ++p1) {
    const int rows = (int)c_binom.v[nb][p1];
    if (p1 >= 2) {
      // phase A: row pairs (a1, s1 ^ a1), a1 not in {0, s1}; G lanes per row,
      // the level's rows x G lanes in passes of TPI (one pass up to m = 13)
      const int g = batch_rows_g(p1);
      const int G = 1 << g;
      for (int pass = 0; pass < (rows << g); pass += TPI) {
        const int ri = (pass + t) >> g;
        const uint32_t r = (uint32_t)t & (uint32_t)(G - 1);
        uint32_t acc[kBRow];
#pragma unroll
        for (int i = 0; i < kBRow; ++i) acc[i] = 0xFFFFFFFFu;
        if (ri < rows) {
          const uint32_t s1 = colex_unrank((unsigned long long)ri, p1, nb);
          const uint32_t lowb = s1 & (~s1 + 1u);
          uint32_t hi = 0, rr = s1;
          for (int q = 0; q < g; ++q) {
            const uint32_t top = 1u << (31 - __clz(rr));
            hi |= top;
            rr ^= top;
          }
          const uint32_t freem = s1 ^ hi;
          const uint32_t fixed = deposit_bits(r, hi);
          uint32_t sub = 0;
          do {
            const uint32_t a1 = fixed | sub;
            if (a1 != 0 && a1 != s1) {
              uint32_t x[kBRow], y[kBRow];
              bload_row(x, Gp + brow_pos(a1) * kBRowStride);
              bload_row(y, Gp + brow_pos(s1 ^ a1) * kBRowStride);
              const uint32_t yb = (s1 ^ a1) << 5;
#pragma unroll
              for (int i = 0; i < kBRow; ++i) y[i] -= yb | (uint32_t)i;  // Gc = Gp - X
              bconv_restricted(acc, x, y);
              if (a1 & lowb) acc[0] = min(acc[0], x[0] + y[0]);
            }
            sub = (sub - freem) & freem;
          } while (sub != 0);
        }
        for (int off = G >> 1; off > 0; off >>= 1) {
#pragma unroll
          for (int i = 0; i < kBRow; ++i) acc[i] = min(acc[i], __shfl_xor_sync(0xFFFFFFFFu, acc[i], off));
        }
        if (ri < rows && r == 0) {
#pragma unroll
          for (int i = 0; i < kBRow; ++i) bk[ri * kBkStride + i] = acc[i];
        }
      }
      __syncthreads();
    }
    // phase B: one thread finishes each row of the level (one pass up to
    // m = 15, passes of TPI rows at m = 16)
    for (int rb = 0; rb < (kGRows ? rows : 1); rb += TPI) {
    const int tr = rb + t;
      if (tr < rows) {
        const uint32_t s1 = colex_unrank((unsigned long long)tr, p1, nb);
        const uint32_t S1 = s1 << 5;
        uint32_t* prow = Gp + brow_pos(s1) * kBRowStride;
        uint32_t zp[kBRow], zcs[kBRow], cc[kBRow];
        bload_row(zp, Gp);   // row 0 is at position 0
        bload_row(zcs, Gp);
#pragma unroll
        for (int i = 0; i < kBRow; ++i) zcs[i] += S1 - (uint32_t)i;  // Gc(0, x) + (s1 << 5): the A-part of a1 = s1 splits
#pragma unroll
        for (int blk = 0; blk < kBRow / 8; ++blk) {
          uint32_t wv[8], bkv[8];
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            wv[q] = prow[blk * 8 + q];
            bkv[q] = p1 >= 2 ? bk[tr * kBkStride + blk * 8 + q] : 0xFFFFFFFFu;
          }
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const int s2 = blk * 8 + q;
            uint32_t f, A;
            if (s2 == 0 && p1 == 1) {  // U = (s1, 0) is a single request
              f = wv[q];
              A = 0;
            } else {
              // two independent minima (a1 = 0 and a1 = s1) shorten the chains
              uint32_t k0 = bkv[q], k1 = 0xFFFFFFFFu;
              if (s2 != 0) {
#pragma unroll
                for (int a2 = 1; a2 < kBRow; ++a2) {
                  if ((a2 & s2) == a2 && (a2 & (s2 & -s2)) != 0) {
                    k0 = min(k0, zp[a2] + cc[s2 ^ a2]);                             // a1 = 0
                    if (a2 != s2) k1 = min(k1, cc[a2] + zcs[s2 ^ a2] + (uint32_t)a2);  // a1 = s1
                  }
                }
              }
              const uint32_t key = min(k0, k1);
              f = (key >> m) - wv[q];
              A = key & mask;
            }
            cc[s2] = f << m;
            put_split(S1 | (uint32_t)s2, A, &bflags);
          }
        }
        uint32_t gp[kBRow];
#pragma unroll
        for (int i = 0; i < kBRow; ++i) gp[i] = cc[i] + (S1 | (uint32_t)i);
        bstore_row(prow, gp);
      }
    }
    __syncthreads();
  }

  // outputs: tables and OPT
  if (use_off) {
    __shared__ long long hi_off[batch_rows_hi_entries(TPI, kGRows)];
    for (int i = t; i < (N + TPI - 1) / TPI; i += TPI)
      hi_off[i] = batch_pi((uint32_t)i * TPI, off) + (long long)off[kBatchUniv];
    __syncthreads();
    const int64_t lo = batch_pi((uint32_t)t & (TPI - 1), off);
    for (int U = t; U < N; U += TPI) {
      F_out[tb + U] = (int64_t)(Gp[bidx((uint32_t)U)] >> m) + batch_offset<TPI>((uint32_t)U, lo, hi_off);
      if (!gsplit) split_out[tb + U] = split[U];
    }
    if (t == 0) opt_out[inst] = (int64_t)(Gp[bidx(mask)] >> m) + batch_pi(mask, off) + (int64_t)off[kBatchUniv];
  } else {
    for (int U = t; U < N; U += TPI) {
      F_out[tb + U] = (int64_t)(Gp[bidx((uint32_t)U)] >> m);
      if (!gsplit) split_out[tb + U] = split[U];
    }
    if (t == 0) opt_out[inst] = (int64_t)(Gp[bidx(mask)] >> m);
  }
  __syncthreads();
  if (gsplit)
    batch_walk<TPI>(inst, m, r0, o0, roff, static_cast<const uint32_t*>(gsp), keys, cx, cN, nd, perm_out, dfs_out,
                    status);
  else
    batch_walk<TPI>(inst, m, r0, o0, roff, split, keys, cx, cN, nd, perm_out, dfs_out, status);
  if (kBoundsChecked) {
    __syncthreads();
    if (t == 0 && bflags) status[inst] = bflags;
  }
}

}  // namespace

size_t batch_smem_bytes(int max_m, int occ_cap) {
  return (size_t)occ_cap * 8 + ((size_t)4 << max_m) + ((size_t)2 << max_m) + (size_t)occ_cap * 8 +
         (size_t)occ_cap * 8 + 64;
}

// One grid over `count` instances of size m (ids inst_list[0..count)).
cudaError_t launch_batch(int count, int m, int occ_cap, const int64_t* weights, const int64_t* inst_req,
                         const int64_t* req_off, const int64_t* chunks, const int64_t* tab_off,
                         const int32_t* inst_list, const uint8_t* flags, int64_t* opt, int64_t* F,
                         uint32_t* split, int64_t* perm, int32_t* dfs, int32_t* status, cudaStream_t stream) {
  const size_t smem = batch_smem_bytes(m, occ_cap);
  cudaError_t e = cudaFuncSetAttribute(k_batch_solve, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k_batch_solve<<<(unsigned)count, kBatchThreads, smem, stream>>>(weights, inst_req, req_off, chunks, tab_off,
                                                                  inst_list, flags, occ_cap, m, opt, F, split,
                                                                  perm, dfs, status);
  return cudaGetLastError();
}

size_t batch_rows_smem_bytes(int m, int occ_cap) {
  const size_t R = (size_t)1 << (m - 5);
  return (m >= kBGlobalRowsM ? 0 : R * kBRowStride * 4) + (size_t)batch_level_rows(m - 5) * kBkStride * 4 +
         (size_t)occ_cap * 16 + (size_t)occ_cap * 8 + (m >= kBGlobalSplitM ? 0 : ((size_t)2 << m)) + 64;
}

// 4-byte words of global row scratch one instance of size m needs (0 while
// its rows fit shared memory)
size_t batch_rows_scratch_words(int m) {
  return m >= kBGlobalRowsM ? ((size_t)1 << (m - 5)) * kBRowStride : 0;
}

// One grid of the row-blocked kernel over `count` instances of size m >= 6
// whose request weights allow packed keys.
cudaError_t launch_batch_rows(int count, int m, int occ_cap, const int64_t* weights, const int64_t* inst_req,
                              const int64_t* req_off, const int64_t* chunks, const int64_t* tab_off,
                              const int32_t* inst_list, const uint8_t* flags, int64_t* opt, int64_t* F,
                              uint32_t* split, int64_t* perm, int32_t* dfs, int32_t* status, uint32_t* rows_scratch,
                              cudaStream_t stream) {
  if (m < 6 || m > kBMaxRowsM || (m >= kBGlobalRowsM && !rows_scratch)) return cudaErrorInvalidValue;
  const size_t smem = batch_rows_smem_bytes(m, occ_cap);
  const int tpi = batch_rows_threads(m);
  cudaError_t e = cudaSuccess;
  auto go = [&](auto kernel) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e == cudaSuccess)
      kernel<<<(unsigned)count, tpi, smem, stream>>>(weights, inst_req, req_off, chunks, tab_off, inst_list, flags,
                                                      occ_cap, m, opt, F, split, perm, dfs, status, rows_scratch);
  };
  if (m >= kBGlobalRowsM)
    go(k_batch_rows<256, true>);
  else if (tpi == 64)
    go(k_batch_rows<64>);
  else if (tpi == 128)
    go(k_batch_rows<128>);
  else
    go(k_batch_rows<256>);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace mpt
