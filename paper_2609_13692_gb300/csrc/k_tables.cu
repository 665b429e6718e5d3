// Natural-order views of the blocked path's tables.
//
// The blocked recurrence (k_dp_blocked.cu) keeps every table in rotated
// order, idx(S) = (T << b) | U with T = S mod 2^L and U = S >> L, so that the
// 2^b subsets of one tile are contiguous.  The natural order S = (U << L) | T
// is the transpose of that 2^L x 2^b matrix; it is produced only when the
// tables themselves are asked for, by a shared-memory tiled transpose (32 x 32
// tiles: reads coalesced along U, writes along T).  The same pass adds back
// the weights that the blocked recurrence leaves out (k_scatter_zeta.cu):
// the private pi_i and the universal u, i.e. sum_{i in S} pi_i + u to F(S)
// for non-empty S, u to every w(I(S)), plus pi_i at S = {i} and sum_i pi_i at
// S = {}, the weight of the union of all requests.
#include "mpt_internal.cuh"

namespace mpt {
namespace {

constexpr int kTile = 32;
constexpr int kRowsPerPass = 8;

struct Copy {
  template <typename S>
  __device__ static S apply(S v, int) { return v; }
};
struct GpToF {
  __device__ static uint32_t apply(uint32_t v, int b) { return v >> b; }
};
struct Gp64ToF {
  __device__ static unsigned long long apply(unsigned long long v, int b) { return v >> b; }
};

enum Offset { kNone, kPiOfS, kPiOfSingletons };

// dst[(U << L) | T] = Op(src[(T << b) | U]) + offset(S) for T < 2^L, U < 2^b,
// S = (U << L) | T: offset pi(S) + u for S non-empty (F), or u plus pi_i at
// S = {i} and sum_i pi_i at S = {} (w(I)), or none; priv null means no
// offsets.
template <typename Src, typename Dst, typename Op, Offset Off>
__global__ void __launch_bounds__(kTile * kRowsPerPass)
k_unrotate(const Src* __restrict__ src, Dst* __restrict__ dst, int L, int b,
           const unsigned long long* __restrict__ priv, int m) {
  __shared__ Dst t[kTile][kTile + 1];
  __shared__ long long piT[kTile], piU[kTile], pi_all, univ;
  const size_t nT = (size_t)1 << L, nU = (size_t)1 << b;
  const size_t T0 = (size_t)blockIdx.x * kTile, U0 = (size_t)blockIdx.y * kTile;
  const int tx = threadIdx.x, ty = threadIdx.y;
  if (Off != kNone && ty < 3) {
    // row 0: pi of the block's T values (requests 0..L-1), row 1: of its U
    // values (requests L..m-1), row 2, lane 0: of all requests
    long long v = 0;
    const size_t x = (ty == 0 ? T0 : U0) + tx;
    if (priv && ty < 2 && x < (ty == 0 ? nT : nU)) {
      for (uint32_t r = (uint32_t)x; r; r &= r - 1) v += (long long)priv[(ty == 0 ? 0 : L) + __ffs(r) - 1];
    }
    if (ty == 0) piT[tx] = v;
    if (ty == 1) piU[tx] = v;
    if (ty == 2 && tx == 0) {
      v = 0;
      if (priv)
        for (int i = 0; i < m; ++i) v += (long long)priv[i];
      pi_all = v;
      univ = priv ? (long long)priv[kUniversalSlot] : 0;
    }
  }
#pragma unroll
  for (int j = 0; j < kTile; j += kRowsPerPass) {
    const size_t T = T0 + ty + j, U = U0 + tx;
    if (T < nT && U < nU) t[ty + j][tx] = (Dst)Op::apply(src[(T << b) | U], b);
  }
  __syncthreads();
#pragma unroll
  for (int j = 0; j < kTile; j += kRowsPerPass) {
    const size_t U = U0 + ty + j, T = T0 + tx;
    if (T < nT && U < nU) {
      Dst v = t[tx][ty + j];
      const uint32_t S = ((uint32_t)U << L) | (uint32_t)T;
      if (Off == kPiOfS) {
        if (S != 0) v += (Dst)(piT[tx] + piU[ty + j] + univ);
      } else if (Off == kPiOfSingletons) {
        v += (Dst)univ;
        if (S == 0)
          v += (Dst)pi_all;
        else if ((S & (S - 1)) == 0)
          v += (Dst)(T ? piT[tx] : piU[ty + j]);
      }
      dst[(U << L) | T] = v;
    }
  }
}

template <typename Src, typename Dst, typename Op, Offset Off>
cudaError_t unrotate(const Src* src, Dst* dst, const Shape& s, const unsigned long long* priv, cudaStream_t stream) {
  const dim3 grid((unsigned)((((size_t)1 << s.L) + kTile - 1) / kTile),
                  (unsigned)((((size_t)1 << s.b) + kTile - 1) / kTile));
  k_unrotate<Src, Dst, Op, Off><<<grid, dim3(kTile, kRowsPerPass), 0, stream>>>(src, dst, s.L, s.b, priv, s.m);
  return cudaGetLastError();
}

}  // namespace

cudaError_t unrotate_tables(const Shape& s, const uint32_t* split_rot, uint32_t* split_nat, const int64_t* wI_rot,
                            int64_t* wI_nat, const uint32_t* Gp, int64_t* F_nat, int32_t* F32_nat,
                            const unsigned long long* priv, cudaStream_t stream) {
  cudaError_t e = cudaSuccess;
  if (split_nat && (e = unrotate<uint32_t, uint32_t, Copy, kNone>(split_rot, split_nat, s, nullptr, stream)) !=
                       cudaSuccess)
    return e;
  if (wI_nat && (e = unrotate<int64_t, int64_t, Copy, kPiOfSingletons>(wI_rot, wI_nat, s, priv, stream)) !=
                    cudaSuccess)
    return e;
  if (F_nat && (e = unrotate<uint32_t, int64_t, GpToF, kPiOfS>(Gp, F_nat, s, priv, stream)) != cudaSuccess) return e;
  if (F32_nat && (e = unrotate<uint32_t, int32_t, GpToF, kPiOfS>(Gp, F32_nat, s, priv, stream)) != cudaSuccess)
    return e;
  return cudaSuccess;
}

cudaError_t unrotate_tables_wide(const Shape& s, const uint32_t* split_rot, uint32_t* split_nat,
                                 const int64_t* wI_rot, int64_t* wI_nat, const unsigned long long* Gp64,
                                 int64_t* F_nat, int32_t* F32_nat, const unsigned long long* priv,
                                 cudaStream_t stream) {
  cudaError_t e = cudaSuccess;
  if (split_nat && (e = unrotate<uint32_t, uint32_t, Copy, kNone>(split_rot, split_nat, s, nullptr, stream)) !=
                       cudaSuccess)
    return e;
  if (wI_nat && (e = unrotate<int64_t, int64_t, Copy, kPiOfSingletons>(wI_rot, wI_nat, s, priv, stream)) !=
                    cudaSuccess)
    return e;
  if (F_nat && (e = unrotate<unsigned long long, int64_t, Gp64ToF, kPiOfS>(Gp64, F_nat, s, priv, stream)) !=
                   cudaSuccess)
    return e;
  if (F32_nat && (e = unrotate<unsigned long long, int32_t, Gp64ToF, kPiOfS>(Gp64, F32_nat, s, priv, stream)) !=
                     cudaSuccess)
    return e;
  return cudaSuccess;
}

}  // namespace mpt
