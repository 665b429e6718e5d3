// Internal declarations shared by the CUDA translation units of libmpt.
// Nothing here is part of the public ABI (include/mpt.h).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cstdlib>

#include <cuda_runtime.h>

#include "../../include/mpt.h"

namespace mpt {

// ---------------------------------------------------------------------------
// Binomial coefficients C(n, k), n, k <= 32, for ranking k-subsets in colex
// order (the combinatorial number system): the subset {c_1 < .. < c_k} has
// rank sum_t C(c_t, t).  Every translation unit gets its own constant copy.
// ---------------------------------------------------------------------------
struct BinomTable {
  unsigned long long v[33][33];
};

constexpr BinomTable make_binom() {
  BinomTable t{};
  for (int n = 0; n <= 32; ++n)
    for (int k = 0; k <= 32; ++k)
      t.v[n][k] = (k == 0) ? 1ull : (n == 0 ? 0ull : t.v[n - 1][k - 1] + t.v[n - 1][k]);
  return t;
}

static __constant__ BinomTable c_binom = make_binom();
static constexpr BinomTable h_binom = make_binom();

// The idx-th k-subset of {0..n-1} in colex order.
__device__ __forceinline__ uint32_t colex_unrank(unsigned long long idx, int k, int n) {
  uint32_t S = 0;
  for (int pos = n - 1; pos >= 0 && k > 0; --pos) {
    unsigned long long c = c_binom.v[pos][k];
    if (idx >= c) {
      S |= 1u << pos;
      idx -= c;
      --k;
    }
  }
  return S;
}

// Rank of S among the subsets of its size, in colex order.
__device__ __forceinline__ uint32_t colex_rank(uint32_t S) {
  uint32_t r = 0;
  int t = 1;
  while (S) {
    int pos = __ffs(S) - 1;
    r += (uint32_t)c_binom.v[pos][t];
    ++t;
    S &= S - 1;
  }
  return r;
}

// Scatter the low bits of q into the set positions of mask (ascending).
__device__ __forceinline__ uint32_t deposit_bits(uint32_t q, uint32_t mask) {
  uint32_t out = 0;
  while (mask && q) {
    uint32_t low = mask & (~mask + 1u);
    if (q & 1u) out |= low;
    q >>= 1;
    mask ^= low;
  }
  return out;
}

// ---------------------------------------------------------------------------
// Device-side error flags (bitwise OR into one int in the workspace).
// ---------------------------------------------------------------------------
enum DeviceError : int {
  kErrBadSplit = 1,      // a split entry on the hierarchy is not a proper non-empty subset
  kErrLayoutCount = 2,   // the layout walk did not place every chunk occurrence
  kErrWorkspace = 4,     // a kernel saw a size outside what the workspace was carved for
  kErrTimeout = 8,       // a bounded wait on a shared-memory barrier gave up
  kErrBounds = 16,       // bounds-checked build: an index, window offset or split failed its check
};

// Bounds-checked build (-DMPT_BOUNDS; build(bounds=True)), the stand-in for a
// memory checker: kernels test table indices, window offsets and split
// entries, record kErrBounds in the device flags (mpt_solve then returns
// MPT_ERR_INTERNAL) and skip the access.  In the default build MPT_BAD is
// the constant false and every check compiles away.
#ifdef MPT_BOUNDS
#define MPT_BAD(flags, ok) (!(ok) && (atomicOr((flags), ::mpt::kErrBounds), true))
constexpr bool kBoundsChecked = true;
#else
#define MPT_BAD(flags, ok) false
constexpr bool kBoundsChecked = false;
#endif

// A split entry A of subset S (natural order) is well formed when S has at
// most one request and A = 0, or A is a proper non-empty part of S that
// holds S's lowest request (the Sec. 3.1 recurrence under the tie reading).
__host__ __device__ __forceinline__ bool valid_split(uint32_t S, uint32_t A) {
  if ((S & (S - 1u)) == 0) return A == 0;
  return (A & ~S) == 0 && (A & S & (~S + 1u)) != 0 && A != S;
}

// ---------------------------------------------------------------------------
// Shared-memory barriers (mbarrier) and bulk global -> shared copies.  Every
// wait is bounded: after kWaitTries polls it gives up and reports false, and
// the caller flags kErrTimeout instead of spinning on.
// ---------------------------------------------------------------------------
constexpr uint32_t kWaitTries = 1u << 24;

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(unsigned long long* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

// Make the initialised barriers visible to the copy engine (the async proxy).
__device__ __forceinline__ void mbar_init_fence() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(unsigned long long* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(unsigned long long* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(unsigned long long* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return done != 0;
}

// Wait until the barrier's phase with this parity has completed; false if it
// did not within kWaitTries polls.
__device__ __forceinline__ bool mbar_wait(unsigned long long* bar, uint32_t parity) {
  for (uint32_t i = 0; i < kWaitTries; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

// One contiguous global -> shared copy by the copy engine; its bytes count
// against the barrier's expected transaction bytes.  Both addresses 16-byte
// aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_copy_g2s(void* smem_dst, const void* gmem_src, uint32_t bytes,
                                              unsigned long long* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(smem_u32(smem_dst)), "l"(gmem_src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// ---------------------------------------------------------------------------
// Streaming multiprocessors of the current device, for the grid caps of
// grid-stride loops (a host query of a few microseconds; 152 on a GB300,
// also returned if the query fails, in which case the launch that follows
// reports the error).
// ---------------------------------------------------------------------------
inline int64_t sm_count() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      sms < 1)
    return 152;
  return sms;
}

// ---------------------------------------------------------------------------
// Device allocation of the library's own buffers.  Setting
// MPT_FAIL_DEVICE_ALLOC=1 in the environment makes it fail as an exhausted
// device would (cudaErrorMemoryAllocation), before any CUDA call, so that the
// out-of-memory path of every entry point can be tested on any machine.
// ---------------------------------------------------------------------------
inline cudaError_t device_alloc(void** p, size_t bytes) {
  const char* f = std::getenv("MPT_FAIL_DEVICE_ALLOC");
  if (f && f[0] == '1') return cudaErrorMemoryAllocation;
  return cudaMalloc(p, bytes);
}

// ---------------------------------------------------------------------------
// Workspace carve-up (all offsets 256-byte aligned).
// ---------------------------------------------------------------------------
constexpr int kOffsetSlots = 33;

// Per-instance flags of a batch (mpt_batch.cu, k_batch.cu): packed 32-bit keys,
// and private / universal chunks kept out of the keys.
constexpr uint8_t kFlagPacked = 1;
constexpr uint8_t kFlagOffsets = 2;
constexpr int kUniversalSlot = 32;

struct Workspace {
  // inputs
  int64_t* weights;   // [n]
  uint64_t* bits;     // [m * words]
  // scatter outputs
  uint32_t* used_N;   // [slots]  request set N_x of each used chunk
  int32_t* used_x;    // [slots]  chunk id
  int32_t* counters;  // [8]      0: number of used chunks, 1: device error flags
  // tables, natural subset order (int64 tables: wI and F; lean: fw alone,
  // w(I(S)) until the recurrence writes F(S) over it).  The blocked path
  // leaves them in rotated order (below) and fills the natural views only
  // when they are asked for (unrotate_tables).
  int64_t* wI;        // [2^m] or nullptr
  int64_t* F;         // [2^m] or nullptr
  int32_t* fw;        // [2^m] (lean) or nullptr
  uint32_t* split;    // [2^m]
  // blocked DP working tables, rotated order idx(S) = (T << b) | U with
  // T = S mod 2^L and U = S >> L (see k_dp_blocked.cu)
  uint32_t* Gp;       // [2^m]  F' << b, F'(S) = F(S) - sum_{i in S} pi_i - u
  uint32_t* Gc;       // [2^m]  (F' << b) | (~u & (2^b - 1))
  unsigned long long* partial;  // [max tiles of one layer << b]
  // wide blocked path (64-bit keys): Gp and Gc hold uint64 entries, and the
  // pair kernel leaves one (key, Ta) slot of 2^b entries per block
  unsigned long long* Gp64;     // [2^m] or nullptr
  unsigned long long* Gc64;     // [2^m] or nullptr
  uint32_t* partial_ta;         // [partial_entries] (wide) or nullptr
  int64_t* wI_rot;    // [2^m] w(I(S)) at idx(S) (int64 tables), or nullptr
  int32_t* fw_rot;    // [2^m] w(I(S)) at idx(S) (lean tables), or nullptr
  uint32_t* split_rot;  // [2^m] split[S] at idx(S)
  // blocked paths: slot i < 32 holds pi_i, the weight of the chunks that
  // request i alone needs, and slot kUniversalSlot the weight u of the
  // chunks that every request needs (m >= 2); K1 adds those chunks here
  // instead of to g, and the rotated tables hold w(I) and F less them (see
  // the scatter in k_scatter_zeta.cu)
  unsigned long long* priv;  // [kOffsetSlots] or nullptr
  // layout
  unsigned long long* keys;  // [slots]
  int64_t* perm_offsets;     // [m + 1]
  int64_t* perm_chunks;      // [slots]
  int32_t* dfs;              // [m]
  int64_t* opt;              // [1]
};

struct Shape {
  int m;
  int64_t n;
  int64_t words;
  int64_t slots;    // sum_i |R_i|
  bool blocked;     // blocked DP tables present
  bool wide;        // blocked path with 64-bit keys (shared weight >= 2^(32-b))
  bool lean;        // one int32 table for w(I(S)) then F(S)
  int b;            // tile bits (blocked)
  int L;            // m - b
  int64_t partial_entries;
};

size_t carve_workspace(const Shape& s, char* base, Workspace* ws);

// Rotated position of subset S in the blocked path's tables.
__host__ __device__ __forceinline__ size_t rot_index(uint32_t S, int L, int b) {
  return ((size_t)(S & ((1u << L) - 1u)) << b) | (size_t)(S >> L);
}

// The table K1 scatters into and K2 transforms: w(I) in rotated order for the
// blocked path, natural order for the general one.
inline void* g_table(const Shape& s, const Workspace& ws) {
  if (s.lean) return s.blocked ? (void*)ws.fw_rot : (void*)ws.fw;
  return s.blocked ? (void*)ws.wI_rot : (void*)ws.wI;
}

// ---------------------------------------------------------------------------
// Launchers.  All enqueue on `stream` and return the launch error (if any).
// ---------------------------------------------------------------------------
cudaError_t launch_scatter(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches);
cudaError_t launch_zeta(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches);

// The recurrence runs in steps that depend only on earlier steps: the blocked
// path has one step per tile layer |T| = 0..L, the general path one for the
// singletons and one per popcount layer 2..m.  Launchers run steps
// [step_begin, step_end) (step_end < 0: to the last).
int dp_steps(const Shape& s);
cudaError_t launch_dp_general(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches,
                              int step_begin = 0, int step_end = -1);

struct BlockedTiming {
  cudaEvent_t* pair_ev;  // 2 per pair-kernel launch (start, stop), or nullptr
  cudaEvent_t* tile_ev;  // 2 per tile-kernel launch, or nullptr
  int pair_launches;
  int tile_launches;
  double pair_splits;
};
int blocked_max_launches(const Shape& s);  // upper bound on pair + tile launches
cudaError_t launch_dp_blocked(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches,
                              BlockedTiming* timing, int step_begin = 0, int step_end = -1);
int64_t blocked_partial_entries(int m, int b);
int blocked_tile_bits(int m);

// Pair ranges per tile for one pair-kernel layer (whole waves of one block
// per SM; see k_dp_blocked.cu); at most max_items.
void choose_items(unsigned long long tiles, uint32_t P, int sms, unsigned long long max_items,
                  unsigned long long* items, uint32_t* ppi);

// Wide blocked path (k_dp_wide.cu): 64-bit keys, valid when the shared
// weight sum_i (w(R_i) - pi_i) is below 2^51.  Partial slots: blocks of one
// pair layer, at most.
int64_t wide_partial_slots(int m, int b);
cudaError_t launch_dp_wide(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches,
                           BlockedTiming* timing, int step_begin = 0, int step_end = -1);

cudaError_t launch_walk(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches);

// Natural-order tables from the blocked path's rotated ones (k_tables.cu):
// split_nat[S] = split_rot[idx(S)]; wI_nat[S] = wI_rot[idx(S)] + u plus
// pi_i for S = {i} and sum_i pi_i for S = {} (int64 tables); F_nat[S] or
// F32_nat[S] = (Gp[idx(S)] >> b) + sum_{i in S} pi_i + u (S non-empty).
// priv (the kOffsetSlots offsets on the device) may be null: no offsets.  Null destinations are skipped; they run
// in this order, so a destination may be the source of an earlier conversion.
cudaError_t unrotate_tables(const Shape& s, const uint32_t* split_rot, uint32_t* split_nat, const int64_t* wI_rot,
                            int64_t* wI_nat, const uint32_t* Gp, int64_t* F_nat, int32_t* F32_nat,
                            const unsigned long long* priv, cudaStream_t stream);
// The same for the wide path (F from the uint64 Gp table).
cudaError_t unrotate_tables_wide(const Shape& s, const uint32_t* split_rot, uint32_t* split_nat,
                                 const int64_t* wI_rot, int64_t* wI_nat, const unsigned long long* Gp64,
                                 int64_t* F_nat, int32_t* F32_nat, const unsigned long long* priv,
                                 cudaStream_t stream);
// eq. (1) for any number of strings by lexicographic sorting (k_sched.cu)
mpt_status trie_cost_lex(const int64_t* weights, int64_t n_chunks, int64_t m, const int64_t* offsets,
                         const int64_t* chunks, cudaStream_t st, int64_t* cost);
cudaError_t launch_trie_cost(int m, const int64_t* d_weights, const int64_t* d_offsets, const int64_t* d_chunks,
                             int64_t* d_cost, cudaStream_t stream);

}  // namespace mpt
