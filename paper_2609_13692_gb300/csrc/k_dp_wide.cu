// K3, wide blocked form: the Sec. 3.1 recurrence
//     F({i}) = w(R_i),   F(S) = min over S = A (+) B of F(A) + F(B) - w(I(S)),
// with the tiling of k_dp_blocked.cu (rotated tables, tile T and inner U,
// proper pairs per window pair, the self pair inside the tile) and 64-bit
// packed keys, for instances whose candidate sums do not fit the 32-bit keys
// (shared weight sum_i w(R_i) - sum_i pi_i - m u >= 2^(32-b), F and w(I) less
// the offsets of k_scatter_zeta.cu) but stay below 2^51:
//     key = Gp[A] + Gc[B] = ((F(A) + F(B)) << b) | (2^b - 1 - U + Ua),
// Gp = F << b and Gc = Gp | (~u & (2^b - 1)) as uint64.  The candidates and
// the tie order (value, Ua, Ta) are those of the 32-bit path, so the argmin is
// the same: the least A as an integer among the optimal splits.
//
// Pair kernel.  Windows of 4096 uint64 entries are 256 rows of 16, padded to
// 18 words and XOR-placed.  A unit (s1, a1) is one 4-bit register
// convolution (81 add-min steps) of row a1 of X with row s1 ^ a1 of Y into
// the 16 outputs of row s1.  The 3^8 = 6561 units of a window pair come in
// 1645 chunks (the units of one row with fixed low bits: 4, or 1-2 for the
// rows with fewer than 2 bits), cut into 256 ranges of 7 or 6 consecutive
// chunks; warps 0..3 run the 7-chunk ranges and warps 4..7 the others, so
// each sub-partition issues 13 chunk-times per pair for 12.85 of work.  A thread
// keeps one row's 16 minima in registers while its chunks stay in that row,
// and merges them into a per-pair shared array (64-bit atomicMin) when the
// row changes.  Owners fold the array into running (key, Ta) bests after
// every pair (pairs in increasing Ta, strict improvement), and each block
// writes its 4096 bests to a slot of its own: no atomics in global memory.
//
// Tile kernel.  One block per tile finishes all 4096 entries level by level
// in |U|: the self pair (A = (T, Ua), B = (0, U \ Ua)) or, for tile 0, the
// whole recurrence over the inner bits, by lanes per subset, then the
// lexicographic (key, Ta) minimum with the tile's pair slots.
#include "mpt_internal.cuh"

namespace mpt {
namespace {

using u64 = unsigned long long;

constexpr int kWB = 12;                   // inner bits
constexpr int kWB2 = 4;                   // inner bits held in registers
constexpr int kWB1 = kWB - kWB2;          // 8 row bits
constexpr int kWRow = 1 << kWB2;          // 16 entries per row
constexpr int kWRowStride = kWRow + 2;    // 18 words (144 bytes): XOR-placed rows start in distinct bank groups
constexpr int kWRows = 1 << kWB1;         // 256 rows
constexpr int kWWin = kWRows * kWRowStride;
constexpr int kWThreads = 256;
constexpr int kWOwned = (1 << kWB) / kWThreads;  // 16 outputs folded per thread
constexpr int kWSmemBytes = (2 * 2 * kWWin + 2 * (1 << kWB)) * (int)sizeof(u64);
constexpr int kWTileThreads = 512;
constexpr int kWTileSmemBytes = 2 * (1 << kWB) * (int)sizeof(u64) + (1 << kWB) * (int)sizeof(uint16_t);
constexpr int kWChunks = 1645;
constexpr int kWLong = 109;               // threads with 7 chunks; the others take 6

static_assert(kWLong * 7 + (kWThreads - kWLong) * 6 == kWChunks, "chunk split");
static_assert(kWSmemBytes <= 227 * 1024 && kWTileSmemBytes <= 227 * 1024, "shared memory");

constexpr int popc8(uint32_t v) {
  int c = 0;
  while (v) {
    v &= v - 1;
    ++c;
  }
  return c;
}

constexpr uint32_t deposit8(uint32_t q, uint32_t mask) {
  uint32_t out = 0;
  while (mask) {
    const uint32_t lowb = mask & (~mask + 1u);
    if (q & 1u) out |= lowb;
    q >>= 1;
    mask ^= lowb;
  }
  return out;
}

struct WidePlan {
  uint32_t chunk[kWChunks];          // s1 | fixed << 8 | free << 16
  uint16_t first[kWThreads];         // thread t runs chunks first[t] .. first[t] + count[t] - 1
  uint16_t count[kWThreads];
  int nchunk, total;
};

// Chunks in increasing row order.  Rows with >= 2 bits: the two highest bits
// are free (4 units in Gray order), the others fixed; a 1-bit row is one
// chunk of 2 units, row 0 one chunk of 1 unit.
constexpr WidePlan make_wide_plan() {
  WidePlan pl{};
  int n = 0;
  for (uint32_t s1 = 0; s1 < (uint32_t)kWRows; ++s1) {
    const int p = popc8(s1);
    if (p < 2) {
      pl.chunk[n++] = s1 | (s1 << 16);
      continue;
    }
    uint32_t top = 0, r = s1;
    for (int t = 0; t < 2; ++t) {
      uint32_t hb = 0;
      for (int bit = kWB1 - 1; bit >= 0; --bit)
        if ((r >> bit) & 1u) {
          hb = 1u << bit;
          break;
        }
      top |= hb;
      r ^= hb;
    }
    const uint32_t lowm = s1 ^ top;
    for (uint32_t v = 0; v < (1u << (p - 2)); ++v) pl.chunk[n++] = s1 | (deposit8(v, lowm) << 8) | (top << 16);
  }
  pl.nchunk = n;
  // Ranges r = 0..255 of consecutive chunks, 7 for r < 109 and 6 after.  Lane
  // l of warp w runs range 4 l + w (warps 0..3) or 128 + 4 l + (w - 4): the
  // 7-chunk ranges stay on warps 0..3, and neighbouring lanes work 4 ranges
  // (about 26 chunks) apart, mostly in different rows, so their flushes do
  // not hit the same words.
  int firsts[kWThreads] = {};
  int c = 0;
  for (int r = 0; r < kWThreads; ++r) {
    firsts[r] = c;
    c += r < kWLong ? 7 : 6;
  }
  pl.total = c;
  for (int t = 0; t < kWThreads; ++t) {
    const int w = t / 32, l = t % 32;
    const int r = w < 4 ? 4 * l + w : 128 + 4 * l + (w - 4);
    pl.first[t] = (uint16_t)firsts[r];
    pl.count[t] = (uint16_t)(r < kWLong ? 7 : 6);
  }
  return pl;
}

constexpr WidePlan kWidePlanHost = make_wide_plan();
static_assert(kWidePlanHost.nchunk == kWChunks && kWidePlanHost.total == kWChunks, "chunk plan");
static __constant__ WidePlan c_wplan = make_wide_plan();

// The 4096 subsets of 12 inner bits sorted by size, then colex rank: the order
// in which the tile kernel finishes them.  The same for every tile, so it is
// a static table (global memory, read with coalesced loads) rather than being
// recomputed per block from the binomial table, whose per-thread indices the
// constant cache would serve one by one.
struct OrderTable {
  uint16_t v[1 << kWB];
};

constexpr OrderTable make_order12() {
  OrderTable t{};
  uint32_t start[kWB + 2] = {};
  for (int p = 0; p <= kWB; ++p) start[p + 1] = start[p] + (uint32_t)h_binom.v[kWB][p];
  for (uint32_t u = 0; u < (1u << kWB); ++u) {
    uint32_t r = 0, s = u;
    int k = 1;
    while (s) {
      int pos = 0;
      while (!((s >> pos) & 1u)) ++pos;
      r += (uint32_t)h_binom.v[pos][k];
      ++k;
      s &= s - 1;
    }
    t.v[start[popc8(u)] + r] = (uint16_t)u;
  }
  return t;
}

static __device__ const OrderTable g_order12 = make_order12();

// Row placement: the low 3 row bits XOR-ed with higher ones; linear over GF(2).
__device__ __forceinline__ uint32_t row_pos_w(uint32_t r) { return r ^ (((r >> 3) ^ (r >> 6)) & 7u); }

__device__ __forceinline__ void cp_async16_w(void* smem_dst, const void* gmem_src) {
  const uint32_t d = (uint32_t)__cvta_generic_to_shared(smem_dst);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async_commit_w() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_w() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

// Copy the two windows of a pair: thread t moves the 16-byte chunks t + 256 j
// (j < 8) of each window, i.e. rows (t >> 3) + 32 j, column t & 7.
__device__ __forceinline__ void stage_pair_w(u64* X, u64* Y, const u64* __restrict__ gx, const u64* __restrict__ gy) {
  const uint32_t t = threadIdx.x;
  const uint32_t rp0 = row_pos_w(t >> 3);
  const uint32_t col = (t & 7u) * 2u;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const uint32_t d = (rp0 ^ row_pos_w((uint32_t)(32 * j))) * kWRowStride + col;
    cp_async16_w(X + d, gx + 2 * (t + (uint32_t)(kWThreads * j)));
    cp_async16_w(Y + d, gy + 2 * (t + (uint32_t)(kWThreads * j)));
  }
}

__device__ __forceinline__ void load_row_w(u64 (&v)[kWRow], const u64* p) {
  const ulonglong2* q = reinterpret_cast<const ulonglong2*>(p);
#pragma unroll
  for (int c = 0; c < kWRow / 2; ++c) {
    const ulonglong2 t = q[c];
    v[2 * c] = t.x;
    v[2 * c + 1] = t.y;
  }
}

// acc[s2] = min(acc[s2], min over a2 in s2 of x[a2] + y[s2 ^ a2])  (81 steps)
__device__ __forceinline__ void conv16(u64 (&acc)[kWRow], const u64 (&x)[kWRow], const u64 (&y)[kWRow]) {
#pragma unroll
  for (int a2 = 0; a2 < kWRow; ++a2) {
#pragma unroll
    for (int s2 = 0; s2 < kWRow; ++s2) {
      if ((a2 & s2) == a2) {
        const u64 c = x[a2] + y[s2 ^ a2];
        acc[s2] = c < acc[s2] ? c : acc[s2];
      }
    }
  }
}

__global__ void __launch_bounds__(kWThreads, 1)
k_dp_pairs_w(const u64* __restrict__ Gp, const u64* __restrict__ Gc, u64* __restrict__ pkey, uint32_t* __restrict__ pta,
             int L, int kh, uint32_t pairs_per_tile, uint32_t items_per_tile, uint32_t pairs_per_item,
             int32_t* __restrict__ flags) {
  extern __shared__ __align__(16) u64 wsm[];
  u64* pmin = wsm + 4 * kWWin;  // two per-pair minimum arrays of 4096

  const uint32_t tile = blockIdx.x / items_per_tile;
  const uint32_t item = blockIdx.x % items_per_tile;
  const uint32_t T = colex_unrank(tile, kh, L);
  const uint32_t low = T & (~T + 1u);
  const uint32_t R = T ^ low;
  const uint32_t q0 = item * pairs_per_item;
  const uint32_t q1 = min(q0 + pairs_per_item, pairs_per_tile);
#ifdef MPT_BOUNDS
  {
    // the tile, and every pair's Ta: a proper part of T holding its lowest
    // request, so both windows lie inside the tables
    bool good = tile < c_binom.v[L][kh] && T < (1u << L) && __popc(T) == kh && q1 <= pairs_per_tile;
    uint32_t sb = deposit_bits(q0, R);
    for (uint32_t q = q0; q < q1 && good; ++q) {
      const uint32_t Ta = low | sb;
      good = (Ta & ~T) == 0 && Ta != T;
      sb = (sb - R) & R;
    }
    if (MPT_BAD(flags, good)) return;  // the same decision in every thread
  }
#endif
  // this thread's chunks, read from constant memory once (lanes read
  // different entries, which the constant cache serves one at a time)
  const uint32_t c0 = c_wplan.first[threadIdx.x];
  const int nch = (int)c_wplan.count[threadIdx.x];
  uint32_t chunks[7];
#pragma unroll
  for (int i = 0; i < 7; ++i) chunks[i] = i < nch ? c_wplan.chunk[c0 + i] : 0u;

  for (int i = threadIdx.x; i < 2 * (1 << kWB); i += kWThreads) pmin[i] = ~0ull;
  u64 bk[kWOwned];
  uint32_t bt[kWOwned];
#pragma unroll
  for (int j = 0; j < kWOwned; ++j) {
    bk[j] = ~0ull;
    bt[j] = 0;
  }

  uint32_t sub = deposit_bits(q0, R);
  {
    const uint32_t Ta = low | sub;
    stage_pair_w(wsm, wsm + kWWin, Gp + ((size_t)Ta << kWB), Gc + ((size_t)(T ^ Ta) << kWB));
    cp_async_commit_w();
  }
  for (uint32_t q = q0; q < q1; ++q) {
    const int cur = (int)((q - q0) & 1u);
    const uint32_t Ta = low | sub;
    const uint32_t next = (sub - R) & R;
    if (q + 1 < q1) {
      const uint32_t Tn = low | next;
      u64* nb = wsm + 2 * (cur ^ 1) * kWWin;
      stage_pair_w(nb, nb + kWWin, Gp + ((size_t)Tn << kWB), Gc + ((size_t)(T ^ Tn) << kWB));
      cp_async_commit_w();
      cp_async_wait_w<1>();
    } else {
      cp_async_wait_w<0>();
    }
    __syncthreads();
    const u64* X = wsm + 2 * cur * kWWin;
    const u64* Y = X + kWWin;
    u64* pm = pmin + cur * (1 << kWB);
    {
      uint32_t row = 0xFFFFFFFFu;
      u64 acc[kWRow];
#pragma unroll
      for (int i = 0; i < kWRow; ++i) acc[i] = ~0ull;
#pragma unroll
      for (int c = 0; c < 7; ++c) {
        if (c >= nch) break;
        const uint32_t ch = chunks[c];
        const uint32_t s1 = ch & 0xFFu, fixed = (ch >> 8) & 0xFFu, freem = (ch >> 16) & 0xFFu;
        if (s1 != row) {
          if (row != 0xFFFFFFFFu) {
#pragma unroll
            for (int i = 0; i < kWRow; ++i) atomicMin(&pm[(row << kWB2) | (uint32_t)i], acc[i]);
          }
          row = s1;
#pragma unroll
          for (int i = 0; i < kWRow; ++i) acc[i] = ~0ull;
        }
        const uint32_t ps1 = row_pos_w(s1);
        const uint32_t b0 = freem & (~freem + 1u), b1 = freem ^ b0;
        const int nunits = freem == 0 ? 1 : (b1 == 0 ? 2 : 4);
        uint32_t pa = row_pos_w(fixed);
#pragma unroll 1
        for (int k = 0; k < nunits; ++k) {
          // Gray order over the free bits: fixed, ^b0, ^b1, ^b0
          if (k > 0) pa ^= row_pos_w((k & 1) ? b0 : b1);
          u64 x[kWRow], y[kWRow];
          load_row_w(x, X + pa * kWRowStride);
          load_row_w(y, Y + (pa ^ ps1) * kWRowStride);
          conv16(acc, x, y);
        }
      }
      if (row != 0xFFFFFFFFu) {
#pragma unroll
        for (int i = 0; i < kWRow; ++i) atomicMin(&pm[(row << kWB2) | (uint32_t)i], acc[i]);
      }
    }
    __syncthreads();
    // fold this pair's minima into the running bests; reset the array for the
    // pair after next
#pragma unroll
    for (int j = 0; j < kWOwned; ++j) {
      const uint32_t o = threadIdx.x + (uint32_t)(j * kWThreads);
      const u64 v = pm[o];
      pm[o] = ~0ull;
      if (v < bk[j]) {
        bk[j] = v;
        bt[j] = Ta;
      }
    }
    sub = next;
  }

  const size_t slot = (size_t)blockIdx.x << kWB;
#pragma unroll
  for (int j = 0; j < kWOwned; ++j) {
    const uint32_t o = threadIdx.x + (uint32_t)(j * kWThreads);
    pkey[slot + o] = bk[j];
    pta[slot + o] = bt[j];
  }
}

template <typename Tab>
__device__ __forceinline__ int64_t load_wI_w(const Tab* p) {
  return (int64_t)__ldg(p);
}

// Tile kernel (any |T| = kh, any b <= 12): finishes the tile's 2^b entries.
template <typename Tab>
__global__ void __launch_bounds__(kWTileThreads)
k_dp_tile_w(int L, int b, int kh, const Tab* __restrict__ wIr, const u64* __restrict__ pkey,
            const uint32_t* __restrict__ pta, uint32_t items, u64* __restrict__ Gp, u64* __restrict__ Gc,
            uint32_t* __restrict__ split_rot, int32_t* __restrict__ flags) {
  extern __shared__ __align__(16) u64 tsm[];
  u64* cur = tsm;                       // this tile, F << b
  u64* oc = tsm + (1 << kWB);           // complement form: this tile (kh = 0) or tile 0 (kh >= 1)
  uint16_t* order = reinterpret_cast<uint16_t*>(tsm + 2 * (1 << kWB));  // subsets by size, then colex

  const uint32_t tile = blockIdx.x;
  const uint32_t T = kh == 0 ? 0u : colex_unrank(tile, kh, L);
  const int size = 1 << b;
  const uint32_t mask = (uint32_t)size - 1u;

  for (int u = threadIdx.x; u < size; u += kWTileThreads) {
    if (b == kWB) {
      order[u] = g_order12.v[u];
    } else {  // fewer than 12 requests: tile 0 only, one block
      const int p = __popc(u);
      uint32_t start = 0;
      for (int j = 0; j < p; ++j) start += (uint32_t)c_binom.v[b][j];
      order[start + colex_rank((uint32_t)u)] = (uint16_t)u;
    }
    if (kh >= 1) oc[u] = Gc[u];
  }
  __syncthreads();

  uint32_t start = 0;
  for (int p = 0; p <= b; ++p) {
    const int cnt = (int)c_binom.v[b][p];
    const int g = p > 3 ? min(p - 3, 5) : 0;  // log2(lanes per output)
    const int G = 1 << g;
    const int groups = kWTileThreads >> g;
    for (int base = 0; base < cnt; base += groups) {
      const int gi = base + (int)(threadIdx.x >> g);
      const uint32_t r = threadIdx.x & (uint32_t)(G - 1);
      const bool active = gi < cnt;
      u64 best = ~0ull;
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
          uint32_t s = 0;
          do {
            const uint32_t part = fixed | s;
            if (part != emask) {
              const uint32_t Ua = lowU | part;
              const u64 key = cur[Ua] + oc[U ^ Ua];
              best = key < best ? key : best;
            }
            s = (s - freem) & freem;
          } while (s != 0);
        }
      }
      // the self pair's candidates carry Ta = T (kh = 0: none); the pair
      // kernel's slots of this tile, one per block, are spread over the G
      // lanes of the output; then the lexicographic (key, Ta) minimum of the
      // group, in which the self pair wins ties only against larger Ta
      uint32_t ta = kh == 0 ? 0u : T;
      if (active && kh >= 2) {
        for (uint32_t it = r; it < items; it += (uint32_t)G) {
          const size_t w = ((size_t)(tile * items + it) << b) | U;
          const u64 k2 = pkey[w];
          const uint32_t t2 = pta[w];
          if (k2 < best || (k2 == best && t2 < ta)) {
            best = k2;
            ta = t2;
          }
        }
      }
      for (int off = G >> 1; off > 0; off >>= 1) {
        const u64 o = __shfl_xor_sync(0xFFFFFFFFu, best, off);
        const uint32_t ot = __shfl_xor_sync(0xFFFFFFFFu, ta, off);
        if (o < best || (o == best && ot < ta)) {
          best = o;
          ta = ot;
        }
      }
      if (active && r == 0) {
        const size_t idx = ((size_t)T << b) | U;
        int64_t f;
        uint32_t A;
        if (U == 0 && T == 0) {
          f = 0;
          A = 0;
        } else if (single) {
          f = load_wI_w(wIr + idx);
          A = 0;
        } else {
          const uint32_t Ua = (uint32_t)(best & mask) + U - mask;
          f = (int64_t)(best >> b) - load_wI_w(wIr + idx);
          A = (Ua << L) | ta;
        }
        const u64 gp = (u64)f << b;
        const u64 gc = gp | (u64)(~U & mask);
        cur[U] = gp;
        if (kh == 0) oc[U] = gc;
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

}  // namespace

int64_t wide_partial_slots(int m, int b) {
  const int L = m - b;
  unsigned long long most = 0;
  for (int k = 2; k <= L; ++k)
    if (h_binom.v[L][k] > most) most = h_binom.v[L][k];
  return most > 0 ? (int64_t)(2 * most) : 1;
}

cudaError_t launch_dp_wide(const Shape& s, const Workspace& ws, cudaStream_t stream, int* launches,
                           BlockedTiming* timing, int step_begin, int step_end) {
  cudaError_t e = cudaFuncSetAttribute(k_dp_pairs_w, cudaFuncAttributeMaxDynamicSharedMemorySize, kWSmemBytes);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_dp_tile_w<int64_t>, cudaFuncAttributeMaxDynamicSharedMemorySize, kWTileSmemBytes);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_dp_tile_w<int32_t>, cudaFuncAttributeMaxDynamicSharedMemorySize, kWTileSmemBytes);
  if (e != cudaSuccess) return e;
  int sms = 0, dev = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;

  const int b = s.b, L = s.L;
  const unsigned long long slots = (unsigned long long)wide_partial_slots(s.m, b);
  constexpr unsigned long long evals_per_pair = 531441ull;
  if (step_end < 0 || step_end > L + 1) step_end = L + 1;
  for (int kh = step_begin < 0 ? 0 : step_begin; kh < step_end; ++kh) {
    const unsigned long long tiles = h_binom.v[L][kh];
    unsigned long long items = 0;
    if (kh >= 2) {
      const uint32_t P = (1u << (kh - 1)) - 1u;
      uint32_t ppi = P;
      const unsigned long long max_items = slots / tiles > 0 ? slots / tiles : 1;
      choose_items(tiles, P, sms, max_items, &items, &ppi);
      if (timing && timing->pair_ev) cudaEventRecord(timing->pair_ev[2 * timing->pair_launches], stream);
      k_dp_pairs_w<<<(unsigned)(tiles * items), kWThreads, kWSmemBytes, stream>>>(
          ws.Gp64, ws.Gc64, ws.partial, ws.partial_ta, L, kh, P, (uint32_t)items, ppi, ws.counters + 1);
      if (timing && timing->pair_ev) cudaEventRecord(timing->pair_ev[2 * timing->pair_launches + 1], stream);
      if (timing) {
        timing->pair_launches++;
        timing->pair_splits += (double)tiles * (double)P * (double)evals_per_pair;
      }
      ++*launches;
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    if (timing && timing->tile_ev) cudaEventRecord(timing->tile_ev[2 * timing->tile_launches], stream);
    const unsigned grid = kh == 0 ? 1u : (unsigned)tiles;
    if (s.lean)
      k_dp_tile_w<<<grid, kWTileThreads, kWTileSmemBytes, stream>>>(L, b, kh, ws.fw_rot, ws.partial, ws.partial_ta,
                                                                     (uint32_t)items, ws.Gp64, ws.Gc64, ws.split_rot,
                                                                     ws.counters + 1);
    else
      k_dp_tile_w<<<grid, kWTileThreads, kWTileSmemBytes, stream>>>(L, b, kh, ws.wI_rot, ws.partial, ws.partial_ta,
                                                                     (uint32_t)items, ws.Gp64, ws.Gc64, ws.split_rot,
                                                                     ws.counters + 1);
    if (timing && timing->tile_ev) cudaEventRecord(timing->tile_ev[2 * timing->tile_launches + 1], stream);
    if (timing) timing->tile_launches++;
    ++*launches;
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace mpt
