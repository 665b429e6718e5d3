// mpt_solve_noalloc: the exact solve for callers that cannot allocate device
// memory (see include/mpt.h).  Its scratch -- the blocked recurrence's two
// working tables, the per-layer minima and a few counters -- lives in one
// file-scope device array that every GPU loading this library keeps until
// the process exits.  Nothing here calls cudaMalloc, cudaFree or any
// allocating routine; the kernels are the same ones mpt_solve launches.
#include <cstring>
#include <mutex>

#include "../../include/mpt.h"
#include "mpt_internal.cuh"

namespace {

constexpr int kNoAllocMaxM = 20;          // largest request count accepted
constexpr int kNoAllocTileBits = 12;      // inner bits of the blocked kernels at m >= 12
constexpr int64_t kNoAllocMaxSlots = 1 << 16;  // largest sum of request sizes accepted
constexpr size_t kAlign = 256;

constexpr size_t align_up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

constexpr size_t max_partial_entries() {
  // largest C(L, k) with L = kNoAllocMaxM - 12, times 2^12 inner subsets
  size_t best = 0;
  const int L = kNoAllocMaxM - kNoAllocTileBits;
  for (int k = 0; k <= L; ++k) {
    size_t c = 1;
    for (int j = 0; j < k; ++j) c = c * (size_t)(L - j) / (size_t)(j + 1);
    if (c > best) best = c;
  }
  return best << kNoAllocTileBits;
}

// carve-up of the scratch array
constexpr size_t kOffCounters = 0;
constexpr size_t kOffUsedN = align_up(kOffCounters + 8 * sizeof(int32_t));
constexpr size_t kOffUsedX = align_up(kOffUsedN + kNoAllocMaxSlots * sizeof(uint32_t));
constexpr size_t kOffGp = align_up(kOffUsedX + kNoAllocMaxSlots * sizeof(int32_t));
constexpr size_t kOffGc = align_up(kOffGp + (sizeof(uint32_t) << kNoAllocMaxM));
constexpr size_t kOffPartial = align_up(kOffGc + (sizeof(uint32_t) << kNoAllocMaxM));
constexpr size_t kOffCheck = align_up(kOffPartial + max_partial_entries() * sizeof(unsigned long long));
constexpr int kChecks = 8;
constexpr size_t kOffPriv = align_up(kOffCheck + kChecks * sizeof(unsigned long long));
constexpr size_t kScratchBytes = align_up(kOffPriv + mpt::kOffsetSlots * sizeof(unsigned long long));

// The scratch: about 10.7 MiB per device.  In host code `g_noalloc_scratch`
// is only a host-side stand-in for the symbol; kernels receive the device
// address obtained from cudaGetSymbolAddress below.
__device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
char* g_scratch_ptr[kMaxDevices] = {};
int g_sm_count[kMaxDevices] = {};

// Per-device set-up: the device address of the scratch array and the SM
// count of the current device, looked up once and cached (so a
// cudaDeviceReset while the library is loaded leaves a stale address).
cudaError_t scratch_for_current_device(char** out, int* sms) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_ptr[dev]) {
    int count = 0;
    e = cudaDeviceGetAttribute(&count, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_sm_count[dev] = count > 0 ? count : 1;
    g_scratch_ptr[dev] = static_cast<char*>(p);
  }
  *out = g_scratch_ptr[dev];
  *sms = g_sm_count[dev];
  return cudaSuccess;
}

// Argument checks that need the device-resident inputs: every weight >= 1,
// no request bit at a chunk >= n, the number of chunk occurrences,
// sum_i w(R_i), and the request weight of the chunks that one request alone
// or (m >= 2) every request needs (left out of the blocked recurrence's keys,
// see k_scatter_zeta.cu).  Each
// term w(x) * |S_x| is capped at 2^62 (beyond which the instance is rejected
// anyway) and added as two 32-bit halves into separate 64-bit counters, which
// cannot wrap for n < 2^31.
//   check[0] = bad weight or stray bit, check[1] = occurrences,
//   check[2] / check[3] = sums of the low / high halves of the terms,
//   check[4] / check[5] = the same for the private chunks' terms,
//   check[6] / check[7] = the same for the universal chunks' terms
__global__ void k_noalloc_check(const int64_t* __restrict__ w, const uint64_t* __restrict__ bits, int64_t n, int m,
                                int64_t words, unsigned long long* __restrict__ check) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < words * 64; x += stride) {
    const int64_t word = x >> 6;
    const int sh = (int)(x & 63);
    int cnt = 0;
    for (int i = 0; i < m; ++i) cnt += (int)((bits[(int64_t)i * words + word] >> sh) & 1ull);
    if (x >= n) {
      if (cnt) atomicOr(&check[0], 1ull);
      continue;
    }
    const int64_t wx = w[x];
    if (wx <= 0) {
      atomicOr(&check[0], 1ull);
      continue;
    }
    if (cnt) {
      atomicAdd(&check[1], (unsigned long long)cnt);
      const unsigned long long cap = 1ull << 62;
      const unsigned long long term =
          (unsigned long long)wx > cap / (unsigned long long)cnt ? cap : (unsigned long long)wx * (unsigned long long)cnt;
      atomicAdd(&check[2], term & 0xFFFFFFFFull);
      atomicAdd(&check[3], term >> 32);
      if (cnt == 1) {
        atomicAdd(&check[4], term & 0xFFFFFFFFull);
        atomicAdd(&check[5], term >> 32);
      } else if (cnt == m) {
        atomicAdd(&check[6], term & 0xFFFFFFFFull);
        atomicAdd(&check[7], term >> 32);
      }
    }
  }
}

}  // namespace

extern "C" mpt_status mpt_solve_noalloc(const int64_t* d_weights, int64_t n_chunks, const uint64_t* d_req_bits,
                                        int32_t m, int64_t* d_F, int64_t* d_wI, uint32_t* d_split, int64_t* d_opt,
                                        void* stream_ptr) {
  if (!d_weights || !d_req_bits || !d_F || !d_wI || !d_split || !d_opt || n_chunks < 1 || n_chunks > INT32_MAX ||
      m < 1)
    return MPT_ERR_INVALID_ARG;
  if (m > kNoAllocMaxM) return MPT_ERR_TOO_LARGE;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_ptr);
  char* base = nullptr;
  int sms = 1;
  if (scratch_for_current_device(&base, &sms) != cudaSuccess) return MPT_ERR_CUDA;

  const int64_t words = (n_chunks + 63) / 64;
  unsigned long long* check = reinterpret_cast<unsigned long long*>(base + kOffCheck);
  if (cudaMemsetAsync(check, 0, kChecks * sizeof(unsigned long long), stream) != cudaSuccess) return MPT_ERR_CUDA;
  {
    int64_t blocks = (words * 64 + 255) / 256;
    if (blocks > (int64_t)sms * 16) blocks = (int64_t)sms * 16;
    k_noalloc_check<<<(unsigned)blocks, 256, 0, stream>>>(d_weights, d_req_bits, n_chunks, m, words, check);
    if (cudaGetLastError() != cudaSuccess) return MPT_ERR_CUDA;
  }
  unsigned long long h_check[kChecks] = {0, 0, 0, 0, 0, 0, 0, 0};
  if (cudaMemcpyAsync(h_check, check, sizeof(h_check), cudaMemcpyDeviceToHost, stream) != cudaSuccess ||
      cudaStreamSynchronize(stream) != cudaSuccess)
    return MPT_ERR_CUDA;
  if (h_check[0]) return MPT_ERR_INVALID_ARG;
  if (h_check[1] > (unsigned long long)kNoAllocMaxSlots) return MPT_ERR_TOO_LARGE;
  const unsigned __int128 sum_w = ((unsigned __int128)h_check[3] << 32) + h_check[2];
  if (sum_w >= ((unsigned __int128)1 << 62)) return MPT_ERR_OVERFLOW;
  const unsigned __int128 private_w = ((unsigned __int128)h_check[5] << 32) + h_check[4] +
                                      ((unsigned __int128)h_check[7] << 32) + h_check[6];

  mpt::Shape s{};
  s.m = m;
  s.n = n_chunks;
  s.words = words;
  s.slots = (int64_t)h_check[1];
  s.b = mpt::blocked_tile_bits(m);
  s.L = m - s.b;
  s.blocked = sum_w - private_w < ((unsigned __int128)1 << (32 - s.b));
  s.partial_entries = s.blocked ? mpt::blocked_partial_entries(m, s.b) : 0;

  mpt::Workspace ws{};
  ws.weights = const_cast<int64_t*>(d_weights);
  ws.bits = const_cast<uint64_t*>(d_req_bits);
  ws.counters = reinterpret_cast<int32_t*>(base + kOffCounters);
  ws.used_N = reinterpret_cast<uint32_t*>(base + kOffUsedN);
  ws.used_x = reinterpret_cast<int32_t*>(base + kOffUsedX);
  ws.wI = d_wI;
  ws.F = d_F;
  ws.split = d_split;
  ws.Gp = reinterpret_cast<uint32_t*>(base + kOffGp);
  ws.Gc = reinterpret_cast<uint32_t*>(base + kOffGc);
  ws.partial = reinterpret_cast<unsigned long long*>(base + kOffPartial);
  ws.priv = s.blocked ? reinterpret_cast<unsigned long long*>(base + kOffPriv) : nullptr;
  // The blocked recurrence works on rotated tables: w(I) in the caller's F
  // table, split in its wI table; the natural outputs are written from them
  // at the end (split, then wI, then F from Gp).
  ws.wI_rot = s.blocked ? d_F : nullptr;
  ws.fw_rot = nullptr;
  ws.split_rot = s.blocked ? reinterpret_cast<uint32_t*>(d_wI) : nullptr;

  // The scratch keeps the previous call's contents: the counters must start
  // at zero, and w(I) is accumulated into (the partial minima are reset by
  // the blocked launcher before each layer; Gp and Gc are fully rewritten).
  int launches = 0;
  if (cudaMemsetAsync(ws.counters, 0, 8 * sizeof(int32_t), stream) != cudaSuccess ||
      cudaMemsetAsync(mpt::g_table(s, ws), 0, sizeof(int64_t) << m, stream) != cudaSuccess ||
      (ws.priv && cudaMemsetAsync(ws.priv, 0, mpt::kOffsetSlots * sizeof(unsigned long long), stream) !=
                      cudaSuccess))
    return MPT_ERR_CUDA;
  if (mpt::launch_scatter(s, ws, stream, &launches) != cudaSuccess) return MPT_ERR_CUDA;
  if (mpt::launch_zeta(s, ws, stream, &launches) != cudaSuccess) return MPT_ERR_CUDA;
  cudaError_t e = s.blocked ? mpt::launch_dp_blocked(s, ws, stream, &launches, nullptr)
                            : mpt::launch_dp_general(s, ws, stream, &launches);
  if (e != cudaSuccess) return MPT_ERR_CUDA;
  if (s.blocked &&
      mpt::unrotate_tables(s, ws.split_rot, d_split, ws.wI_rot, d_wI, ws.Gp, d_F, nullptr, ws.priv, stream) !=
          cudaSuccess)
    return MPT_ERR_CUDA;
  const size_t full = ((size_t)1 << m) - 1;
  if (cudaMemcpyAsync(d_opt, d_F + full, sizeof(int64_t), cudaMemcpyDeviceToDevice, stream) != cudaSuccess)
    return MPT_ERR_CUDA;
  return MPT_OK;
}
