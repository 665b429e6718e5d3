// K3 (blocked form): the Sec. 3.1 recurrence
//     F({i}) = w(R_i),   F(S) = min over S = A (+) B of F(A) + F(B) - w(I(S)),
// evaluated with shared-memory tiles so that each 4-byte table entry fetched
// from HBM/L2 serves hundreds of splits.
//
// Index layout.  Requests are split into a "tile" part T (requests 0..L-1)
// and an "inner" part U (requests L..m-1, b = m - L <= 12 of them).  The
// working tables are stored in rotated order idx(S) = (T << b) | U, so the
// 2^b subsets sharing one T are contiguous (one 16 KB window per T).  The
// w(I) table the kernels read and the split table they write use the same
// order; F itself exists only as Gp = F << b (below).
//
// Split structure.  A split of S = (T, U) is named by its part A = (Ta, Ua)
// that holds the lowest request of S.  For T != 0 that request is in T, so
//   * proper pairs: Ta runs over the subsets of T that hold lowbit(T), Ta != T,
//     and Ua over ALL subsets of U;  B = (T \ Ta, U \ Ua).  For a fixed Ta this
//     is a full min-plus subset convolution over the b inner bits of the two
//     windows F[Ta, .] and F[T \ Ta, .] -- the pair kernel below;
//   * self pair: Ta = T, Ua a proper subset of U, B = (0, U \ Ua): needs the
//     tile's own smaller entries, so it runs inside the tile, level by level
//     in |U| -- the tile kernel below, which also finishes every entry.
// For T = 0 the tile kernel runs the recurrence on the b inner bits alone.
// Tiles with |T| = k depend only on tiles with |T| < k: one launch pair per k.
//
// Packed keys.  The tables hold F less the weight of the chunks that one or
// every request needs (F' of k_scatter_zeta.cu; written F below).  With the
// shared weight sum_i w(R_i) - sum_i pi_i - m u below 2^(32-b) every
// candidate F(A) + F(B) fits in 32 - b bits, so the working tables hold
// G = F << b and the key of a candidate is
//     key = Gp[A] + Gc[B] = ((F(A) + F(B)) << b) | (2^b - 1 - U + Ua),
// Gp = F << b and Gc = (F << b) | (~u & (2^b - 1)) (u = the entry's U part).
// An unsigned min over keys picks the least value and, among equal values,
// the least Ua; across proper pairs, taken in increasing Ta with strict
// improvement, the least Ta; then the self pair (largest Ta = T).  That is the
// lexicographic order on (value, A) as an integer, since A = Ua * 2^L + Ta.
#include "mpt_internal.cuh"

namespace mpt {
namespace {

constexpr int kB = 12;                     // inner bits of the pair kernel
constexpr int kB2 = 5;                     // inner bits held in registers
constexpr int kB1 = kB - kB2;              // inner bits that index window rows
constexpr int kRow = 1 << kB2;             // 32 entries per row
constexpr int kRowStride = kRow + 4;       // 36 words: consecutive rows start in different 16-byte bank groups
constexpr int kRows = 1 << kB1;            // 128 rows per window
constexpr int kWin = kRows * kRowStride;   // words per padded window
constexpr int kPairThreads = 256;         // 8 warps: 2 per SM sub-partition
constexpr int kRing = 4;                   // window-pair slots per block
constexpr int kSharedRows = 34;            // rows merged through shared memory every pair
constexpr int kSharedOut = kSharedRows * kRow;
constexpr int kSharedStride = kRow + 1;    // words per shared row in the per-pair minimum arrays
constexpr int kSharedWords = kSharedRows * kSharedStride;
constexpr int kSharedOwned = (kSharedOut + kPairThreads - 1) / kPairThreads;
constexpr int kExtraUnits = 139;           // shared-row units of one pair
constexpr int kExtraSlots = (kExtraUnits + 31) / 32;  // whole-warp slots per pair: 4 full, 1 of 11 lanes
constexpr int kPartial = kExtraUnits - 32 * (kExtraSlots - 1);  // lanes of the partial slot
constexpr int kPairSmemWords = kRing * 2 * kWin + kRing * kSharedWords + kRow * kPairThreads;
constexpr int kPairSmemBytes = kPairSmemWords * (int)sizeof(uint32_t) + 3 * kRing * 8;
constexpr int kMinPairsPerItem = 16;
constexpr int kTileThreads = 512;
constexpr int kMaxTileBits = 12;

static_assert(kRing * 2 * kWin * (int)sizeof(uint32_t) >= (1 << kB) * 8, "merge buffer must fit in the windows");
static_assert((kRing * 2 * kWin + kRing * kSharedWords + kRow * kPairThreads) % 2 == 0, "8-byte aligned barriers");
static_assert(kExtraSlots == 5 && 2 * kPartial <= 32, "4 full slots per pair; two partial slots fill one warp");
static_assert(kPairThreads == 256, "the slot rotation (9 slots per two pairs over 8 warps) assumes 8 warps");
static_assert((kRowStride * 4) % 16 == 0, "padded rows start on 16-byte boundaries");

// ---------------------------------------------------------------------------
// Work split of the pair kernel.  The b inner bits are (s1, s2): s1 = the top
// kB1 bits (window row), s2 = the low kB2 bits (register lane).  Output
// (s1, s2) collects, for every Ua = (a1, a2) with a1 in s1 and a2 in s2,
// X[a1][a2] + Y[s1^a1][s2^a2].  A "unit" is one (s1, a1): two rows, 243
// add-min steps; row s1 has 2^|s1| units, 3^7 = 2187 in all.
//
// Register rows: every row with >= 3 bits except the first five with exactly
// 3 -- 94 rows, 2048 units -- split on their lowest set bits into 256 tasks of
// exactly 8 units, one per thread.  A thread keeps the 32 outputs of its task
// in registers across all pairs (running best key and Ta), merged with the
// other tasks of the row once, at the end.
// Shared rows: the 29 rows with <= 2 bits and those five -- 34 rows, 139
// units per pair.  They run as whole-warp "slots" of 32 units: 4 full slots
// and one of 11 lanes per pair, the units of one row spread over the slots
// (at most two lanes of a slot flush into one bank; see make_plan).  The
// partial slots of pairs 2h and 2h + 1 run as one slot of 22 lanes, so two
// pairs have 9 slots, numbered 9h .. 9h + 8 and run by warp (number mod 8):
// over 16 pairs every warp runs exactly 9 slots, and each sub-partition 256
// register unit-times plus 18 slots against 273.4 units of work (0.2 % idle
// lanes; 1 % with a partial slot per pair).  A slot's 32 minima go to the
// pair's shared array with atomicMin; owner threads fold that array into
// registers one pair later.
// ---------------------------------------------------------------------------
__host__ __device__ constexpr int popc_c(uint32_t v) {
  int c = 0;
  while (v) {
    v &= v - 1;
    ++c;
  }
  return c;
}

constexpr uint32_t deposit_c(uint32_t q, uint32_t mask) {
  uint32_t out = 0;
  while (mask) {
    const uint32_t low = mask & (~mask + 1u);
    if (q & 1u) out |= low;
    q >>= 1;
    mask ^= low;
  }
  return out;
}

struct PairPlan {
  uint32_t task[kPairThreads];            // s1 | fixed << 8 | free << 16 (8 units)
  uint32_t extra[kExtraSlots * 32];       // s1 | a1 << 8 | shared-row index << 16, or ~0u
  uint32_t srow[kSharedRows];             // s1 of each shared row
  int ntask, nextra, nsrow;
};

constexpr bool is_shared_row(uint32_t s1) {
  const int p = popc_c(s1);
  if (p <= 2) return true;
  if (p != 3) return false;
  int rank = 0;  // the first five 3-bit rows in increasing s1 are shared
  for (uint32_t t = 0; t < s1; ++t)
    if (popc_c(t) == 3) ++rank;
  return rank < 5;
}

constexpr PairPlan make_plan() {
  PairPlan pl{};
  int n = 0, nr = 0, ne = 0;
  for (uint32_t s1 = 0; s1 < (uint32_t)kRows; ++s1) {
    if (is_shared_row(s1)) {
      pl.srow[nr++] = s1;
      continue;
    }
    const int q = popc_c(s1) - 3;
    uint32_t lowbits = 0, r = s1;
    for (int t = 0; t < q; ++t) {
      const uint32_t lb = r & (~r + 1u);
      lowbits |= lb;
      r ^= lb;
    }
    const uint32_t freem = s1 ^ lowbits;
    for (uint32_t v = 0; v < (1u << q); ++v) pl.task[n++] = s1 | (deposit_c(v, lowbits) << 8) | (freem << 16);
  }
  for (int i = 0; i < kExtraSlots * 32; ++i) pl.extra[i] = 0xFFFFFFFFu;
  // Shared-row units are placed so that few lanes of one slot flush into the
  // same bank: rows in decreasing unit count, each unit into the slot that
  // holds the fewest units of rows congruent to its own mod 32 (the bank of
  // word i of shared row r is (r + i) mod 32), then the emptiest slot.
  int fill[kExtraSlots] = {};
  for (int p = kB1; p >= 0; --p) {
    for (int ri = 0; ri < nr; ++ri) {
      const uint32_t s1 = pl.srow[ri];
      if (popc_c(s1) != p) continue;
      for (uint32_t k = 0; k < (1u << p); ++k) {
        int best = -1, best_same = 0, best_room = 0;
        for (int sl = 0; sl < kExtraSlots; ++sl) {
          const int cap = kExtraUnits - 32 * sl < 32 ? kExtraUnits - 32 * sl : 32;
          const int room = cap - fill[sl];
          if (room <= 0) continue;
          int same = 0;
          for (int l = 0; l < fill[sl]; ++l)
            if ((int)((pl.extra[32 * sl + l] >> 16) & 0xFFu) % 32 == ri % 32) ++same;
          if (best < 0 || same < best_same || (same == best_same && room > best_room)) {
            best = sl;
            best_same = same;
            best_room = room;
          }
        }
        const uint32_t a1 = deposit_c(k, s1);
        pl.extra[32 * best + fill[best]++] = s1 | (a1 << 8) | ((uint32_t)ri << 16);
        ++ne;
      }
    }
  }
  pl.ntask = n;
  pl.nextra = ne;
  pl.nsrow = nr;
  return pl;
}

// Largest number of lanes of one slot whose rows share a bank class (rows
// congruent mod 32 put word i in the same bank).
constexpr int max_slot_bank_share(const PairPlan& pl) {
  int worst = 0;
  for (int sl = 0; sl < kExtraSlots; ++sl)
    for (int cls = 0; cls < 32; ++cls) {
      int n = 0;
      for (int l = 0; l < 32; ++l) {
        const uint32_t e = pl.extra[32 * sl + l];
        if (e != 0xFFFFFFFFu && (int)((e >> 16) & 0xFFu) % 32 == cls) ++n;
      }
      worst = n > worst ? n : worst;
    }
  return worst;
}

constexpr PairPlan kPlanHost = make_plan();
static_assert(max_slot_bank_share(kPlanHost) <= 2, "shared-row units spread over the slots");
static_assert(kPlanHost.ntask == kPairThreads, "register tasks must fill the block");
static_assert(kPlanHost.nsrow == kSharedRows, "shared row count");
static_assert(kPlanHost.nextra == kExtraUnits, "extra units");
static __constant__ PairPlan c_plan = make_plan();

// Word of shared output j = (shared row, lane) in a per-pair minimum array:
// rows are 33 words apart, so lanes flushing different rows, and owners
// reading consecutive outputs, hit different banks.
__device__ __forceinline__ uint32_t sw_word(uint32_t j) { return j + (j >> kB2); }

// Row placement inside a padded window: the low 3 row bits are XOR-ed with
// higher row bits so that rows that differ only above bit 2 still start in
// different bank groups.  The map is linear over GF(2):
// row_pos(a ^ b) = row_pos(a) ^ row_pos(b).
__device__ __forceinline__ int row_pos(uint32_t r) { return (int)(r ^ (((r >> 3) ^ (r >> 6)) & 7u)); }

__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gmem_src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(smem_u32(smem_dst)), "l"(gmem_src) : "memory");
}

// Every thread copies its share of the two windows of one pair into a ring
// slot and arms the slot's "full" barrier to count one arrival once those
// copies have landed (the barrier expects one arrival per thread).  Thread t
// copies the 16-byte chunks t + kPairThreads * j: rows (t >> 3) + 32 j of X
// (j < 4) and of Y, always column t & 7.  row_pos is linear, so each chunk's
// padded row position is one XOR away from row_pos(t >> 3).
__device__ __forceinline__ void copy_pair(uint32_t* X, uint32_t* Y, const uint32_t* __restrict__ gx,
                                          const uint32_t* __restrict__ gy, unsigned long long* full) {
  constexpr int kChunks = kRows * kRow / 4;  // 1024 per window
  static_assert(kChunks % kPairThreads == 0, "whole chunks per thread");
  const uint32_t t = threadIdx.x;
  const uint32_t rp0 = (uint32_t)row_pos(t >> 3);
  const uint32_t col = (t & 7u) * 4u;
#pragma unroll
  for (int j = 0; j < kChunks / kPairThreads; ++j) {
    const uint32_t rp = rp0 ^ (uint32_t)row_pos((uint32_t)(j * (kPairThreads / 8)));
    const uint32_t d = rp * kRowStride + col;
    cp_async16(X + d, gx + 4 * (t + (uint32_t)(j * kPairThreads)));
    cp_async16(Y + d, gy + 4 * (t + (uint32_t)(j * kPairThreads)));
  }
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(smem_u32(full)) : "memory");
}

__device__ __forceinline__ void load_row(uint32_t (&v)[kRow], const uint32_t* p) {
  const uint4* q = reinterpret_cast<const uint4*>(p);
#pragma unroll
  for (int c = 0; c < kRow / 4; ++c) {
    const uint4 t = q[c];
    v[4 * c] = t.x;
    v[4 * c + 1] = t.y;
    v[4 * c + 2] = t.z;
    v[4 * c + 3] = t.w;
  }
}

// acc[s2] = min over a2 in s2 of x[a2] + y[s2 ^ a2]  (243 add/min pairs).
// The a2-outer order puts independent accumulators next to each other (an
// order that spreads each accumulator's updates evenly measured 1.7 % slower:
// ptxas schedules this one better).  With kInit the a2 = 0 term initialises
// acc instead of being min-ed into it.
template <bool kInit = false>
__device__ __forceinline__ void conv_rows(uint32_t (&acc)[kRow], const uint32_t (&x)[kRow], const uint32_t (&y)[kRow]) {
#pragma unroll
  for (int a2 = 0; a2 < kRow; ++a2) {
#pragma unroll
    for (int s2 = 0; s2 < kRow; ++s2) {
      if ((a2 & s2) == a2) {
        if (kInit && a2 == 0)
          acc[s2] = x[0] + y[s2];
        else
          acc[s2] = min(acc[s2], x[a2] + y[s2 ^ a2]);
      }
    }
  }
}

// A bounded barrier wait that the whole (converged) warp leaves together:
// true only if every lane saw the phase complete.
__device__ __forceinline__ bool warp_wait(unsigned long long* bar, uint32_t parity) {
  return __all_sync(0xFFFFFFFFu, mbar_wait(bar, parity));
}

// Fold pair jj's shared-row minima (ring slot jj mod kRing) into the running
// bests of the shared outputs this thread owns (a strict improvement takes
// the pair's Ta), reset them for the slot's next pair, and mark the slot
// free.  False if the pair's "consumed" barrier did not complete in time.
__device__ __forceinline__ bool fold_pair(uint32_t jj, uint32_t Ta_jj, uint32_t* smin, unsigned long long* consumed,
                                          unsigned long long* folded, uint32_t (&sbk)[kSharedOwned],
                                          uint32_t (&sbt)[kSharedOwned]) {
  const uint32_t c = jj % kRing;
  if (!warp_wait(&consumed[c], (jj / kRing) & 1u)) return false;
  uint32_t* sm = smin + c * kSharedWords;
#pragma unroll
  for (int j = 0; j < kSharedOwned; ++j) {
    const uint32_t o = threadIdx.x + (uint32_t)(j * kPairThreads);
    if (o < (uint32_t)kSharedOut) {
      const uint32_t w = sw_word(o);
      const uint32_t v = sm[w];
      sm[w] = 0xFFFFFFFFu;
      if (v < sbk[j]) {
        sbk[j] = v;
        sbt[j] = Ta_jj;
      }
    }
  }
  mbar_arrive(&folded[c]);
  return true;
}

// Pair kernel for tiles with |T| = kh >= 2.  Block = (tile, range of pairs).
// Writes, per inner subset U of the tile, the lexicographic minimum of
// (key, Ta) over its pairs into partial[tile << kB | U] with atomicMin.
//
// The pairs of the range stream through a ring of kRing window slots with no
// block-wide barrier.  Pair q lives in slot q mod kRing.  At the start of
// step q every warp waits until all threads have folded pair q + 1 - kRing
// ("folded"), and its threads start their copies of pair q + 1 into that
// slot; then they wait for pair q's copies ("full"), run their slot and
// units, arrive on "consumed", fold the previous pair's shared-row minima
// into their running bests (in pair order) and arrive on "folded".  The warp
// that runs the merged partial slot of pairs q - 1 and q arrives on
// "consumed" of pair q - 1 only after that slot, at step q (before it, no
// thread can fold pair q - 1, whose fold follows the units of step q, and no
// slot of pair q - 1 is refilled).  Every wait is
// bounded; one that gives up sets kErrTimeout in *flags and the thread stops
// (after waiting, bounded again, for the copies it started), so the launch
// ends with its results marked invalid.
__global__ void __launch_bounds__(kPairThreads, 1)
k_dp_pairs(const uint32_t* __restrict__ Gp, const uint32_t* __restrict__ Gc, unsigned long long* __restrict__ partial,
           int L, int kh, uint32_t pairs_per_tile, uint32_t items_per_tile, uint32_t pairs_per_item,
           int32_t* __restrict__ flags) {
  extern __shared__ __align__(16) uint32_t smem[];
  // ring slot c: X at smem + 2c * kWin, Y right after it; then one per-pair
  // minimum array of the shared rows per slot; then the running-best Ta of
  // every register output, [output][thread]; then the barriers
  uint32_t* smin = smem + kRing * 2 * kWin;
  uint32_t* sbest_t = smin + kRing * kSharedWords;
  unsigned long long* full = reinterpret_cast<unsigned long long*>(sbest_t + kRow * kPairThreads);
  unsigned long long* consumed = full + kRing;
  unsigned long long* folded = consumed + kRing;

  const uint32_t tile = blockIdx.x / items_per_tile;
  const uint32_t item = blockIdx.x % items_per_tile;
  const uint32_t T = colex_unrank(tile, kh, L);
  const uint32_t low = T & (~T + 1u);
  const uint32_t R = T ^ low;
  const uint32_t q0 = item * pairs_per_item;
  const uint32_t q1 = min(q0 + pairs_per_item, pairs_per_tile);
  const uint32_t npairs = q1 > q0 ? q1 - q0 : 0u;
  const uint32_t warp = threadIdx.x >> 5, lane = threadIdx.x & 31u;
#ifdef MPT_BOUNDS
  {
    // the tile, and every pair's Ta: a part of T holding its lowest request,
    // so both windows lie inside the 2^(L + kB)-entry tables
    bool good = tile < c_binom.v[L][kh] && T < (1u << L) && __popc(T) == kh && q1 <= pairs_per_tile;
    uint32_t sb = deposit_bits(q0, R);
    for (uint32_t p = 0; p < npairs && good; ++p) {
      const uint32_t Ta = low | sb;
      good = (Ta & ~T) == 0 && Ta != T;
      sb = (sb - R) & R;
    }
    if (MPT_BAD(flags, good)) return;  // the same decision in every thread
  }
#endif

  const uint32_t task = c_plan.task[threadIdx.x];
  const uint32_t s1 = task & 0xFFu;
  const uint32_t fixed = (task >> 8) & 0xFFu;
  const uint32_t freem = (task >> 16) & 0xFFu;  // exactly 3 bits
  const uint32_t b0 = freem & (~freem + 1u);
  const uint32_t b1 = (freem ^ b0) & (~(freem ^ b0) + 1u);
  const uint32_t b2 = freem ^ b0 ^ b1;
  const uint32_t pos_fixed = (uint32_t)row_pos(fixed), pos_s1 = (uint32_t)row_pos(s1);
  const uint32_t pb0 = (uint32_t)row_pos(b0), pb1 = (uint32_t)row_pos(b1), pb2 = (uint32_t)row_pos(b2);
  // this lane's unit in each of the kExtraSlots slots of a pair, and in the
  // merged partial slot (lanes 0..kPartial-1: the earlier pair's partial
  // slot, the next kPartial lanes the later pair's)
  uint32_t ext[kExtraSlots];
#pragma unroll
  for (int i = 0; i < kExtraSlots; ++i) ext[i] = c_plan.extra[32 * i + (int)lane];
  const uint32_t ext_part = __shfl_sync(0xFFFFFFFFu, ext[kExtraSlots - 1], lane < (uint32_t)kPartial ? lane : lane - kPartial);
  const uint32_t ext_merged = lane < 2u * kPartial ? ext_part : 0xFFFFFFFFu;

  if (threadIdx.x == 0) {
    for (int c = 0; c < kRing; ++c) {
      mbar_init(&full[c], kPairThreads);
      mbar_init(&consumed[c], kPairThreads);
      mbar_init(&folded[c], kPairThreads);
    }
    mbar_init_fence();
  }
  for (int i = threadIdx.x; i < kRing * kSharedWords; i += kPairThreads) smin[i] = 0xFFFFFFFFu;
  uint32_t bk[kRow], sbk[kSharedOwned], sbt[kSharedOwned];
#pragma unroll
  for (int i = 0; i < kRow; ++i) {
    bk[i] = 0xFFFFFFFFu;
    sbest_t[i * kPairThreads + threadIdx.x] = 0;
  }
#pragma unroll
  for (int j = 0; j < kSharedOwned; ++j) {
    sbk[j] = 0xFFFFFFFFu;
    sbt[j] = 0;
  }
  __syncthreads();

  // the first pair, into slot 0
  uint32_t sub = deposit_bits(q0, R);
  if (npairs >= 1) copy_pair(smem, smem + kWin, Gp + ((size_t)(low | sub) << kB), Gc + ((size_t)(R ^ sub) << kB), &full[0]);

  bool ok = true;
  uint32_t prev_Ta = 0;
  for (uint32_t j = 0; j < npairs; ++j) {
    const uint32_t c = j % kRing;
    const uint32_t Ta = low | sub;
    const uint32_t next = (sub - R) & R;
    // copies of pair j + 1, into the slot pair j + 1 - kRing has left
    if (j + 1 < npairs) {
      const uint32_t cn = (j + 1) % kRing;
      if (j + 1 >= (uint32_t)kRing && !warp_wait(&folded[cn], (((j + 1) / kRing) - 1u) & 1u)) {
        ok = false;
        break;
      }
      uint32_t* Xn = smem + 2 * cn * kWin;
      copy_pair(Xn, Xn + kWin, Gp + ((size_t)(low | next) << kB), Gc + ((size_t)(R ^ next) << kB), &full[cn]);
    }
    if (!warp_wait(&full[c], (j / kRing) & 1u)) {
      ok = false;
      break;
    }
    const uint32_t* X = smem + 2 * c * kWin;
    const uint32_t* Y = X + kWin;
    {
      uint32_t acc[kRow];
      // This warp's shared-row slot of the step, if the rotation gives it
      // one.  Pairs 2h and 2h + 1 have 9 slots between them, numbered 9h ..
      // 9h + 8 and run by warps (number mod 8): the full slots of pair 2h at
      // step 2h, then those of pair 2h + 1 and the merged partial slot of
      // both at step 2h + 1.  A last pair without a partner runs its own
      // partial slot.  The warp of the merged slot holds back its "consumed"
      // arrival for pair 2h until that slot has flushed.
      const uint32_t h = j >> 1;
      const bool odd = (j & 1u) != 0;
      const uint32_t base = odd ? 9u * h + 4u : 9u * h;
      const uint32_t nslots = odd || j + 1 == npairs ? (uint32_t)kExtraSlots : (uint32_t)kExtraSlots - 1u;
      const uint32_t si = (warp + 8u - base % 8u) % 8u;
      if (si < nslots) {
        uint32_t e = ext[0];
#pragma unroll
        for (int i = 1; i < kExtraSlots; ++i)
          if (si == (uint32_t)i) e = ext[i];
        const bool merged = odd && si == (uint32_t)kExtraSlots - 1u;
        uint32_t cs = c;
        if (merged) {
          e = ext_merged;
          if (lane < (uint32_t)kPartial) cs = (j - 1) % kRing;
        }
        if (e != 0xFFFFFFFFu) {
          const uint32_t es1 = e & 0xFFu, ea1 = (e >> 8) & 0xFFu, erow = (e >> 16) & 0xFFu;
          const uint32_t* Xs = smem + 2 * cs * kWin;
          uint32_t x[kRow], y[kRow];
          load_row(x, Xs + row_pos(ea1) * kRowStride);
          load_row(y, Xs + kWin + row_pos(es1 ^ ea1) * kRowStride);
          conv_rows<true>(acc, x, y);
          uint32_t* row = smin + cs * kSharedWords + erow * kSharedStride;
#pragma unroll
          for (int i = 0; i < kRow; ++i) atomicMin(&row[i], acc[i]);
        }
        if (merged) mbar_arrive(&consumed[(j - 1) % kRing]);
      }
      // The 8 units of the task visit a1 = fixed | sub with sub running over the
      // subsets of its 3 free bits in Gray-code order; row_pos is linear over
      // GF(2), so each step changes the row position by one XOR.
      uint32_t pa = pos_fixed;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (k > 0) pa ^= (k & 1) ? pb0 : ((k & 2) ? pb1 : pb2);
        uint32_t x[kRow], y[kRow];
        load_row(x, X + pa * kRowStride);
        load_row(y, Y + (pa ^ pos_s1) * kRowStride);
        if (k == 0)
          conv_rows<true>(acc, x, y);
        else
          conv_rows(acc, x, y);
      }
#pragma unroll
      for (int i = 0; i < kRow; ++i) {
        bool keep;  // true when the running best is <= this pair's minimum
        bk[i] = __vibmin_u32(bk[i], acc[i], &keep);
        if (!keep) sbest_t[i * kPairThreads + threadIdx.x] = Ta;
      }
    }
    // pair j's arrival, unless this warp runs the merged slot of j and j + 1
    if (!((j & 1u) == 0 && j + 1 < npairs && warp == (j >> 1) % 8u)) mbar_arrive(&consumed[c]);
    if (j >= 1 && !fold_pair(j - 1, prev_Ta, smin, consumed, folded, sbk, sbt)) {
      ok = false;
      break;
    }
    prev_Ta = Ta;
    sub = next;
  }
  if (ok && npairs >= 1) ok = fold_pair(npairs - 1, prev_Ta, smin, consumed, folded, sbk, sbt);
  if (!ok) {
    if (lane == 0) atomicOr(flags, kErrTimeout);
    // the copies this thread started must land before the block's memory goes away
    asm volatile("cp.async.wait_all;" ::: "memory");
  }

  // Merge the threads that share a row, then the blocks that share the tile.
  __syncthreads();
  unsigned long long* merged = reinterpret_cast<unsigned long long*>(smem);
  for (int i = threadIdx.x; i < (1 << kB); i += kPairThreads) merged[i] = ~0ull;
  __syncthreads();
#pragma unroll
  for (int i = 0; i < kRow; ++i)
    atomicMin(&merged[(s1 << kB2) | (uint32_t)i],
              ((unsigned long long)bk[i] << 32) | sbest_t[i * kPairThreads + threadIdx.x]);
#pragma unroll
  for (int jj = 0; jj < kSharedOwned; ++jj) {
    const uint32_t o = threadIdx.x + (uint32_t)(jj * kPairThreads);
    if (o < (uint32_t)kSharedOut) {
      const uint32_t U = (c_plan.srow[o >> kB2] << kB2) | (o & (kRow - 1));
      atomicMin(&merged[U], ((unsigned long long)sbk[jj] << 32) | sbt[jj]);
    }
  }
  __syncthreads();
  unsigned long long* out = partial + ((size_t)tile << kB);
  for (int i = threadIdx.x; i < (1 << kB); i += kPairThreads) atomicMin(&out[i], merged[i]);
}

// Generic tile kernel: finishes every entry of the tiles with |T| = kh, level
// by level in |U|, folding in the self pair (kh >= 1) or running the whole
// recurrence on the inner bits (kh = 0).  One block per tile.  Used for tile 0
// (any b <= 12); the tiles with kh >= 1 go to k_dp_tile_rows.
// Both tile kernels read w(I) and write split in rotated order, one tile's
// entries contiguous; F itself stays in Gp (F << b).
// Tab: int64 w(I) table, or the int32 one of the lean layout.
template <typename Tab>
__device__ __forceinline__ int64_t load_wI(const Tab* p) {
  return (int64_t)__ldg(p);
}

template <typename Tab>
__global__ void __launch_bounds__(kTileThreads)
k_dp_tile(int L, int b, int kh, const Tab* __restrict__ wIr, const unsigned long long* __restrict__ partial,
          uint32_t* __restrict__ Gp, uint32_t* __restrict__ Gc, uint32_t* __restrict__ split_rot,
          int32_t* __restrict__ flags) {
  __shared__ uint32_t cur_p[1 << kMaxTileBits];   // this tile, F << b
  __shared__ uint32_t other_c[1 << kMaxTileBits]; // complement form: this tile (kh = 0) or tile 0 (kh >= 1)
  __shared__ uint16_t order[1 << kMaxTileBits];   // inner subsets sorted by size, then colex

  const uint32_t tile = blockIdx.x;
  const uint32_t T = kh == 0 ? 0u : colex_unrank(tile, kh, L);
  const int size = 1 << b;
  const uint32_t mask = (uint32_t)size - 1u;

  for (int u = threadIdx.x; u < size; u += kTileThreads) {
    const int p = __popc(u);
    uint32_t start = 0;
    for (int j = 0; j < p; ++j) start += (uint32_t)c_binom.v[b][j];
    order[start + colex_rank((uint32_t)u)] = (uint16_t)u;
    if (kh >= 1) other_c[u] = Gc[u];
  }
  __syncthreads();

  uint32_t start = 0;
  for (int p = 0; p <= b; ++p) {
    const int cnt = (int)c_binom.v[b][p];
    const int g = p > 3 ? min(p - 3, 5) : 0;  // log2(lanes per output)
    const int G = 1 << g;
    const int groups = kTileThreads >> g;
    for (int base = 0; base < cnt; base += groups) {
      const int gi = base + (int)(threadIdx.x >> g);
      const uint32_t r = threadIdx.x & (uint32_t)(G - 1);
      const bool active = gi < cnt;
      unsigned long long best = ~0ull;
      uint32_t U = 0;
      bool single = false;
      if (active) {
        U = order[start + gi];
        const uint32_t nreq = (uint32_t)p + (uint32_t)kh;
        single = nreq == 1;
        if (nreq >= 2 && !(kh >= 1 && U == 0)) {
          // kh = 0: Ua = lowbit(U) | part, part a proper subset of U \ lowbit(U).
          // kh >= 1: Ua = part, a proper subset of U (Ta = T).
          const uint32_t lowU = kh == 0 ? (U & (~U + 1u)) : 0u;
          const uint32_t emask = U ^ lowU;
          uint32_t hi = 0, rr = emask;
          for (int t = 0; t < g; ++t) {
            const uint32_t top = 1u << (31 - __clz(rr));
            hi |= top;
            rr ^= top;
          }
          const uint32_t freem = emask ^ hi;
          const uint32_t fixed = deposit_bits(r, hi);
          const unsigned long long ta = kh == 0 ? 0ull : (unsigned long long)T;
          uint32_t s = 0;
          do {
            const uint32_t part = fixed | s;
            if (part != emask) {
              const uint32_t Ua = lowU | part;
              const uint32_t key = cur_p[Ua] + other_c[U ^ Ua];
              const unsigned long long c = ((unsigned long long)key << 32) | ta;
              best = c < best ? c : best;
            }
            s = (s - freem) & freem;
          } while (s != 0);
        }
        if (kh >= 2 && r == 0) {
          const unsigned long long pv = partial[((size_t)tile << b) | U];
          best = pv < best ? pv : best;
        }
      }
      for (int off = G >> 1; off > 0; off >>= 1) {
        const unsigned long long o = __shfl_xor_sync(0xFFFFFFFFu, best, off);
        best = o < best ? o : best;
      }
      if (active && r == 0) {
        const size_t idx = ((size_t)T << b) | U;
        int64_t f;
        uint32_t A;
        if (U == 0 && T == 0) {
          f = 0;
          A = 0;
        } else if (single) {
          f = load_wI(wIr + idx);
          A = 0;
        } else {
          const uint32_t key = (uint32_t)(best >> 32);
          const uint32_t Ua = (key & mask) + U - mask;
          f = (int64_t)(key >> b) - load_wI(wIr + idx);
          A = (Ua << L) | (uint32_t)best;
        }
        const uint32_t gp = (uint32_t)f << b;
        const uint32_t gc = gp | (~U & mask);
        cur_p[U] = gp;
        if (kh == 0) other_c[U] = gc;
        if (!MPT_BAD(flags, idx < ((size_t)1 << (L + b)) && valid_split(T | (U << L), A))) {
          Gp[idx] = gp;
          Gc[idx] = gc;
          split_rot[idx] = A;
        }
      }
    }
    start += (uint32_t)cnt;
    __syncthreads();
  }
}

// Row-blocked tile kernel for |T| = kh >= 1 (inner bits b = kB).  The self
// pair of output U = (s1, s2) has candidates Ua = (a1, a2) with Ua a proper
// subset of U, A = (T, Ua) from this tile and B = (0, U \ Ua) from tile 0:
//   * cross-row: a1 a proper subset of s1, any a2 in s2 -- rows of this tile
//     finished at an earlier popcount level of s1, combined with whole rows of
//     tile 0 by the same register convolution as the pair kernel;
//   * in-row: a1 = s1, a2 a proper subset of s2 -- a 5-bit recurrence inside
//     the row, in registers, in increasing s2 (every proper subset of s2 is
//     smaller than s2).
// Rows are finished level by level in |s1|, so every row read is final.
constexpr int kRowsThreads = 96;
constexpr int kBestWords = (1 << kB) + kRows;  // per-output arrays, rows 33 words apart
// With kZcGlobal, tile 0's complement rows are read from global memory (the
// same 16 KB for every block, so they stay in L1) instead of a shared copy:
// 52 KB of shared memory per block instead of 70, four blocks per SM instead
// of three.  That pays on long layers (m >= 26: 7.95 vs 8.37 ms of tile
// stage at m = 28) but not on short ones (m = 24: 1.22 vs 1.19 ms).
constexpr int rows_smem_bytes(bool zc_global) {
  return ((zc_global ? 1 : 2) * kWin + 2 * kBestWords) * (int)sizeof(uint32_t);
}
constexpr int kZcGlobalMinL = 14;

// Word of output U = (s1, s2) in a per-output array: rows are 33 words apart,
// so threads that hold different rows and the same s2 hit different banks.
__device__ __forceinline__ uint32_t best_word(uint32_t U) { return U + (U >> kB2); }

// Row r of tile 0's complement form (Gc[0 .. 4095] is written by the tile-0
// launch and only read here): from the shared copy, or from global memory.
template <bool kZcGlobal>
__device__ __forceinline__ void load_zrow(uint32_t (&v)[kRow], const uint32_t* zc, const uint32_t* __restrict__ Gc,
                                          uint32_t r) {
  if constexpr (kZcGlobal) {
    const uint4* q = reinterpret_cast<const uint4*>(Gc + r * kRow);
#pragma unroll
    for (int c = 0; c < kRow / 4; ++c) {
      const uint4 t = __ldg(q + c);
      v[4 * c] = t.x;
      v[4 * c + 1] = t.y;
      v[4 * c + 2] = t.z;
      v[4 * c + 3] = t.w;
    }
  } else {
    load_row(v, zc + row_pos(r) * kRowStride);
  }
}

template <typename Tab, bool kZcGlobal>
__global__ void __launch_bounds__(kRowsThreads)
k_dp_tile_rows(int L, int kh, const Tab* __restrict__ wIr, const unsigned long long* __restrict__ partial,
               uint32_t* __restrict__ Gp, uint32_t* __restrict__ Gc, uint32_t* __restrict__ split_rot,
               int32_t* __restrict__ flags) {
  extern __shared__ __align__(16) uint32_t smem[];
  uint32_t* cur = smem;                                   // this tile, F << kB, padded rows
  uint32_t* zc = smem + kWin;                             // tile 0, complement form, padded rows (shared copy)
  uint32_t* bkey = smem + (kZcGlobal ? 1 : 2) * kWin;     // best key per output so far
  uint32_t* bsplit = bkey + kBestWords;                   // its Ta; after finishing, the split A
  constexpr uint32_t kMask = (1u << kB) - 1u;

  const uint32_t tile = blockIdx.x;
  const uint32_t T = colex_unrank(tile, kh, L);
  const size_t tbase = (size_t)T << kB;
  if (MPT_BAD(flags, tile < c_binom.v[L][kh] && T < (1u << L) && __popc(T) == kh)) return;

  if constexpr (!kZcGlobal) {
    for (int c = threadIdx.x; c < (1 << (kB - 2)); c += kRowsThreads) {
      const int row = c >> (kB2 - 2), k = c & ((1 << (kB2 - 2)) - 1);
      *reinterpret_cast<uint4*>(zc + row_pos((uint32_t)row) * kRowStride + 4 * k) =
          *reinterpret_cast<const uint4*>(Gc + 4 * c);
    }
  }
  for (int u = threadIdx.x; u < (1 << kB); u += kRowsThreads) {
    const unsigned long long pv = kh >= 2 ? partial[((size_t)tile << kB) | (uint32_t)u] : ~0ull;
    bkey[best_word((uint32_t)u)] = (uint32_t)(pv >> 32);
    bsplit[best_word((uint32_t)u)] = (uint32_t)pv;
  }
  __syncthreads();

  for (int p1 = 0; p1 <= kB1; ++p1) {
    const int rows = (int)c_binom.v[kB1][p1];
    // The threads that finish this level's rows fetch their w(I(S)) (32
    // consecutive rotated entries each) now, so that the loads complete while
    // phase A runs.
    uint32_t wv[kRow];
    const bool finisher = (int)threadIdx.x < rows;
    const uint32_t s1f = finisher ? colex_unrank((unsigned long long)threadIdx.x, p1, kB1) : 0u;
    if (finisher) {
#pragma unroll
      for (int i = 0; i < kRow; ++i) wv[i] = (uint32_t)load_wI(wIr + (tbase | (s1f << kB2) | (uint32_t)i));
    }
    if (p1 >= 1) {
      // lanes per row chosen so that each lane runs at most 8 row pairs
      const int g = p1 > 3 ? p1 - 3 : 0;
      const int G = 1 << g;
      const int ri = (int)(threadIdx.x >> g);
      const uint32_t r = threadIdx.x & (uint32_t)(G - 1);
      const bool active = ri < rows;
      uint32_t acc[kRow];
#pragma unroll
      for (int i = 0; i < kRow; ++i) acc[i] = 0xFFFFFFFFu;
      uint32_t s1 = 0;
      if (active) {
        s1 = colex_unrank((unsigned long long)ri, p1, kB1);
        uint32_t hi = 0, rr = s1;
        for (int t = 0; t < g; ++t) {
          const uint32_t top = 1u << (31 - __clz(rr));
          hi |= top;
          rr ^= top;
        }
        const uint32_t freem = s1 ^ hi;
        const uint32_t fixed = deposit_bits(r, hi);
        uint32_t sub = 0;
        do {
          const uint32_t a1 = fixed | sub;
          if (a1 != s1) {
            uint32_t x[kRow], y[kRow];
            load_row(x, cur + row_pos(a1) * kRowStride);
            load_zrow<kZcGlobal>(y, zc, Gc, s1 ^ a1);
            conv_rows(acc, x, y);
          }
          sub = (sub - freem) & freem;
        } while (sub != 0);
      }
      for (int off = G >> 1; off > 0; off >>= 1) {
#pragma unroll
        for (int i = 0; i < kRow; ++i) acc[i] = min(acc[i], __shfl_xor_sync(0xFFFFFFFFu, acc[i], off));
      }
      if (active && r == 0) {
#pragma unroll
        for (int i = 0; i < kRow; ++i) {
          const uint32_t U = (s1 << kB2) | (uint32_t)i;
          if (acc[i] < bkey[best_word(U)]) {
            bkey[best_word(U)] = acc[i];
            bsplit[best_word(U)] = T;
          }
        }
      }
      __syncthreads();
    }
    if (finisher) {
      const uint32_t s1 = s1f;
      uint32_t z[kRow], c[kRow];
      load_zrow<kZcGlobal>(z, zc, Gc, 0);
#pragma unroll
      for (int s2 = 0; s2 < kRow; ++s2) {
        uint32_t key = 0xFFFFFFFFu;
#pragma unroll
        for (int a2 = 0; a2 < kRow; ++a2) {
          if ((a2 & s2) == a2 && a2 != s2) key = min(key, c[a2] + z[s2 ^ a2]);
        }
        const uint32_t U = (s1 << kB2) | (uint32_t)s2;
        uint32_t bk = bkey[best_word(U)], bt = bsplit[best_word(U)];
        if (key < bk) {
          bk = key;
          bt = T;
        }
        uint32_t f, A;
        if (kh == 1 && U == 0) {  // S = T, a single request
          f = wv[s2];
          A = 0;
        } else {
          const uint32_t Ua = (bk & kMask) + U - kMask;
          f = (bk >> kB) - wv[s2];
          A = (Ua << L) | bt;
        }
        c[s2] = f << kB;
        bsplit[best_word(U)] = A;
      }
      uint4* dst = reinterpret_cast<uint4*>(cur + row_pos(s1) * kRowStride);
#pragma unroll
      for (int q = 0; q < kRow / 4; ++q) dst[q] = make_uint4(c[4 * q], c[4 * q + 1], c[4 * q + 2], c[4 * q + 3]);
    }
    __syncthreads();
  }

  for (int u = threadIdx.x; u < (1 << kB); u += kRowsThreads) {
    const uint32_t gp = cur[row_pos((uint32_t)u >> kB2) * kRowStride + (u & (kRow - 1))];
    const uint32_t A = bsplit[best_word((uint32_t)u)];
    if (MPT_BAD(flags, valid_split(T | ((uint32_t)u << L), A))) continue;
    Gp[tbase | (uint32_t)u] = gp;
    Gc[tbase | (uint32_t)u] = gp | (~(uint32_t)u & kMask);
    split_rot[tbase | (uint32_t)u] = A;
  }
}

}  // namespace

constexpr unsigned long long kItemOverheadPairs = 2;

// Items (blocks) per tile of one pair-kernel layer.  One block runs per SM,
// every block of a layer takes about the same time per pair, and a block costs
// about kItemOverheadPairs pairs more (its first window copy and its final
// merge).  The layer then takes ceil(blocks / SMs) waves of (pairs per item +
// overhead); take the item count that minimises that, fewer blocks on ties.
// Items keep at least kMinPairsPerItem pairs; at most max_items per tile.
void choose_items(unsigned long long tiles, uint32_t P, int sms, unsigned long long max_items,
                  unsigned long long* items_out, uint32_t* ppi_out) {
  const unsigned long long waves_of = sms > 0 ? (unsigned long long)sms : 1ull;
  unsigned long long cap = (P + kMinPairsPerItem - 1) / kMinPairsPerItem;
  if (cap > max_items) cap = max_items;
  if (cap < 1) cap = 1;
  if (cap > 8192) cap = 8192;
  unsigned long long best_t = ~0ull, best_items = 1;
  uint32_t best_ppi = P;
  for (unsigned long long it = 1; it <= cap; ++it) {
    const uint32_t ppi = (uint32_t)((P + it - 1) / it);
    const unsigned long long items = (P + ppi - 1) / ppi;
    if (items != it) continue;  // the same split as a smaller count
    const unsigned long long waves = (tiles * items + waves_of - 1) / waves_of;
    const unsigned long long t = waves * ((unsigned long long)ppi + kItemOverheadPairs);
    if (t < best_t) {
      best_t = t;
      best_items = items;
      best_ppi = ppi;
    }
  }
  *items_out = best_items;
  *ppi_out = best_ppi;
}

int blocked_tile_bits(int m) { return m < kB ? m : kB; }

int64_t blocked_partial_entries(int m, int b) {
  const int L = m - b;
  unsigned long long most = 0;
  for (int k = 2; k <= L; ++k)
    if (h_binom.v[L][k] > most) most = h_binom.v[L][k];
  return (int64_t)(most << b);
}

int blocked_max_launches(const Shape& s) { return 2 * (s.L + 1); }

cudaError_t launch_dp_blocked(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches,
                              BlockedTiming* timing, int step_begin, int step_end) {
  {
    // the attributes belong to the current device: set them on every call (a
    // host-side call, negligible against a solve), so that any device works
    cudaError_t e = cudaFuncSetAttribute(k_dp_pairs, cudaFuncAttributeMaxDynamicSharedMemorySize, kPairSmemBytes);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k_dp_tile_rows<int64_t, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             rows_smem_bytes(false));
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k_dp_tile_rows<int32_t, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             rows_smem_bytes(false));
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k_dp_tile_rows<int64_t, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             rows_smem_bytes(true));
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k_dp_tile_rows<int32_t, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             rows_smem_bytes(true));
    if (e != cudaSuccess) return e;
  }
  const int b = s.b, L = s.L;
  constexpr unsigned long long evals_per_pair = 531441ull;  // 3^12 splits per pair of windows
  int sms = 0, dev = 0;
  {
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  if (step_end < 0 || step_end > L + 1) step_end = L + 1;
  for (int kh = step_begin < 0 ? 0 : step_begin; kh < step_end; ++kh) {
    const unsigned long long tiles = h_binom.v[L][kh];
    if (kh >= 2) {
      const uint32_t P = (1u << (kh - 1)) - 1u;
      unsigned long long items = 1;
      uint32_t ppi = P;
      choose_items(tiles, P, sms, ~0ull, &items, &ppi);
      cudaError_t e = cudaMemsetAsync(ws.partial, 0xFF, (size_t)(tiles << b) * sizeof(unsigned long long), stream);
      if (e != cudaSuccess) return e;
      if (timing && timing->pair_ev) cudaEventRecord(timing->pair_ev[2 * timing->pair_launches], stream);
      k_dp_pairs<<<(unsigned)(tiles * items), kPairThreads, kPairSmemBytes, stream>>>(
          ws.Gp, ws.Gc, ws.partial, L, kh, P, (uint32_t)items, ppi, ws.counters + 1);
      if (timing && timing->pair_ev) cudaEventRecord(timing->pair_ev[2 * timing->pair_launches + 1], stream);
      if (timing) {
        timing->pair_launches++;
        timing->pair_splits += (double)tiles * (double)P * (double)evals_per_pair;
      }
      ++*launches;
      e = cudaGetLastError();
      if (e != cudaSuccess) return e;
    }
    if (timing && timing->tile_ev) cudaEventRecord(timing->tile_ev[2 * timing->tile_launches], stream);
    if (kh == 0) {
      if (s.lean)
        k_dp_tile<<<1, kTileThreads, 0, stream>>>(L, b, 0, ws.fw_rot, nullptr, ws.Gp, ws.Gc, ws.split_rot,
                                                  ws.counters + 1);
      else
        k_dp_tile<<<1, kTileThreads, 0, stream>>>(L, b, 0, ws.wI_rot, nullptr, ws.Gp, ws.Gc, ws.split_rot,
                                                  ws.counters + 1);
    } else {
      const unsigned long long* part = kh >= 2 ? ws.partial : nullptr;
      const bool zg = L >= kZcGlobalMinL;
      const int sm_bytes = rows_smem_bytes(zg);
      if (s.lean) {
        auto k = zg ? k_dp_tile_rows<int32_t, true> : k_dp_tile_rows<int32_t, false>;
        k<<<(unsigned)tiles, kRowsThreads, sm_bytes, stream>>>(L, kh, ws.fw_rot, part, ws.Gp, ws.Gc, ws.split_rot,
                                                               ws.counters + 1);
      } else {
        auto k = zg ? k_dp_tile_rows<int64_t, true> : k_dp_tile_rows<int64_t, false>;
        k<<<(unsigned)tiles, kRowsThreads, sm_bytes, stream>>>(L, kh, ws.wI_rot, part, ws.Gp, ws.Gc, ws.split_rot,
                                                               ws.counters + 1);
      }
    }
    if (timing && timing->tile_ev) cudaEventRecord(timing->tile_ev[2 * timing->tile_launches + 1], stream);
    if (timing) timing->tile_launches++;
    ++*launches;
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace mpt
