// Natural-order views of the blocked path's tables.
//
// The blocked recurrence (k_dp_blocked.cu) keeps every table in rotated
// order, idx(S) = (T << b) | U with T = S mod 2^L and U = S >> L, so that the
// 2^b subsets of one tile are contiguous.  The natural order S = (U << L) | T
// is the transpose of that 2^L x 2^b matrix; it is produced only when the
// tables themselves are asked for, by a shared-memory tiled transpose (32 x 32
// tiles: reads coalesced along U, writes along T).
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

// dst[(U << L) | T] = Op(src[(T << b) | U]) for T < 2^L, U < 2^b.
template <typename Src, typename Dst, typename Op>
__global__ void __launch_bounds__(kTile * kRowsPerPass)
k_unrotate(const Src* __restrict__ src, Dst* __restrict__ dst, int L, int b) {
  __shared__ Dst t[kTile][kTile + 1];
  const size_t nT = (size_t)1 << L, nU = (size_t)1 << b;
  const size_t T0 = (size_t)blockIdx.x * kTile, U0 = (size_t)blockIdx.y * kTile;
  const int tx = threadIdx.x, ty = threadIdx.y;
#pragma unroll
  for (int j = 0; j < kTile; j += kRowsPerPass) {
    const size_t T = T0 + ty + j, U = U0 + tx;
    if (T < nT && U < nU) t[ty + j][tx] = (Dst)Op::apply(src[(T << b) | U], b);
  }
  __syncthreads();
#pragma unroll
  for (int j = 0; j < kTile; j += kRowsPerPass) {
    const size_t U = U0 + ty + j, T = T0 + tx;
    if (T < nT && U < nU) dst[(U << L) | T] = t[tx][ty + j];
  }
}

template <typename Src, typename Dst, typename Op>
cudaError_t unrotate(const Src* src, Dst* dst, int L, int b, cudaStream_t stream) {
  const dim3 grid((unsigned)((((size_t)1 << L) + kTile - 1) / kTile), (unsigned)((((size_t)1 << b) + kTile - 1) / kTile));
  k_unrotate<Src, Dst, Op><<<grid, dim3(kTile, kRowsPerPass), 0, stream>>>(src, dst, L, b);
  return cudaGetLastError();
}

}  // namespace

cudaError_t unrotate_tables(const Shape& s, const uint32_t* split_rot, uint32_t* split_nat, const int64_t* wI_rot,
                            int64_t* wI_nat, const uint32_t* Gp, int64_t* F_nat, int32_t* F32_nat,
                            cudaStream_t stream) {
  cudaError_t e = cudaSuccess;
  if (split_nat && (e = unrotate<uint32_t, uint32_t, Copy>(split_rot, split_nat, s.L, s.b, stream)) != cudaSuccess)
    return e;
  if (wI_nat && (e = unrotate<int64_t, int64_t, Copy>(wI_rot, wI_nat, s.L, s.b, stream)) != cudaSuccess) return e;
  if (F_nat && (e = unrotate<uint32_t, int64_t, GpToF>(Gp, F_nat, s.L, s.b, stream)) != cudaSuccess) return e;
  if (F32_nat && (e = unrotate<uint32_t, int32_t, GpToF>(Gp, F32_nat, s.L, s.b, stream)) != cudaSuccess) return e;
  return cudaSuccess;
}

cudaError_t unrotate_tables_wide(const Shape& s, const uint32_t* split_rot, uint32_t* split_nat,
                                 const int64_t* wI_rot, int64_t* wI_nat, const unsigned long long* Gp64,
                                 int64_t* F_nat, int32_t* F32_nat, cudaStream_t stream) {
  cudaError_t e = cudaSuccess;
  if (split_nat && (e = unrotate<uint32_t, uint32_t, Copy>(split_rot, split_nat, s.L, s.b, stream)) != cudaSuccess)
    return e;
  if (wI_nat && (e = unrotate<int64_t, int64_t, Copy>(wI_rot, wI_nat, s.L, s.b, stream)) != cudaSuccess) return e;
  if (F_nat && (e = unrotate<unsigned long long, int64_t, Gp64ToF>(Gp64, F_nat, s.L, s.b, stream)) != cudaSuccess)
    return e;
  if (F32_nat && (e = unrotate<unsigned long long, int32_t, Gp64ToF>(Gp64, F32_nat, s.L, s.b, stream)) != cudaSuccess)
    return e;
  return cudaSuccess;
}

}  // namespace mpt
