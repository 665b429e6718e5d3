// C ABI of the batched small-instance solver (include/mpt.h, mpt_batch_*):
// argument checks, workspace carve-up and one grid per instance size m, the
// grids on side streams forked from the caller's stream.
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "../../include/mpt.h"
#include "mpt_internal.cuh"

namespace mpt {
size_t batch_smem_bytes(int max_m, int occ_cap);
size_t batch_rows_smem_bytes(int m, int occ_cap);
size_t batch_rows_scratch_words(int m);
cudaError_t launch_batch(int count, int m, int occ_cap, const int64_t* weights, const int64_t* inst_req,
                         const int64_t* req_off, const int64_t* chunks, const int64_t* tab_off,
                         const int32_t* inst_list, const uint8_t* flags, int64_t* opt, int64_t* F,
                         uint32_t* split, int64_t* perm, int32_t* dfs, int32_t* status, cudaStream_t stream);
cudaError_t launch_batch_rows(int count, int m, int occ_cap, const int64_t* weights, const int64_t* inst_req,
                              const int64_t* req_off, const int64_t* chunks, const int64_t* tab_off,
                              const int32_t* inst_list, const uint8_t* flags, int64_t* opt, int64_t* F,
                              uint32_t* split, int64_t* perm, int32_t* dfs, int32_t* status, uint32_t* rows_scratch,
                              cudaStream_t stream);
}  // namespace mpt

struct mpt_batch {
  int32_t batch = 0;
  int64_t n = 0, requests = 0, occurrences = 0, table_entries = 0;
  int max_m = 0, occ_cap = 1;
  std::vector<int64_t> w, inst_req, req_off, chunks, tab_off;
  // instances grouped by size m: inst_list[group_start[m] .. group_start[m+1]),
  // those for the row-blocked kernel (m >= 6, packed keys) first, up to
  // group_rows_end[m]; each part with its own occurrence cap
  std::vector<int32_t> inst_list;
  std::vector<int64_t> group_start, group_rows_end;
  std::vector<int> group_occ_cap_rows, group_occ_cap;
  // per instance: kFlagPacked when the shared weight is below 2^(32 - m)
  // (32-bit keys), kFlagOffsets when sum_i w(R_i) is not (private and
  // universal chunks kept out of the kernels' values, k_batch.cu)
  std::vector<uint8_t> flags;
  // results of the last solve
  bool solved = false;
  std::vector<int64_t> opt, perm;
  std::vector<int32_t> dfs, status;
  const int64_t* d_F = nullptr;
  const uint32_t* d_split = nullptr;
  void* own_ws = nullptr;
  size_t own_bytes = 0;
  // side streams for the per-size launches (created on first use, on the
  // device current then), with the events that fork them from and join them
  // to the caller's stream
  int side_device = -1;
  std::vector<cudaStream_t> side;
  std::vector<cudaEvent_t> join;
  cudaEvent_t fork = nullptr;
};

namespace {

constexpr int kBatchMaxM = 16;  // m = 16: packed keys only (the row-blocked kernel)
constexpr size_t kBatchMaxSmem = 227 * 1024;  // shared memory of one block
constexpr int kBatchSideStreams = 4;

// Destroys the side streams and events on the device they were made on,
// restoring the caller's current device.
void release_side_streams(mpt_batch* b) {
  int cur = -1;
  const bool switch_dev = b->side_device >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != b->side_device &&
                          cudaSetDevice(b->side_device) == cudaSuccess;
  for (cudaStream_t st : b->side) cudaStreamDestroy(st);
  for (cudaEvent_t ev : b->join) cudaEventDestroy(ev);
  if (b->fork) cudaEventDestroy(b->fork);
  if (switch_dev) cudaSetDevice(cur);
  b->side.clear();
  b->join.clear();
  b->fork = nullptr;
  b->side_device = -1;
}

// The side streams of the current device, created on first use; false when
// they cannot be made (the launches then stay on the caller's stream).
bool side_streams(mpt_batch* b) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  if (b->side_device == dev) return true;
  release_side_streams(b);
  if (cudaEventCreateWithFlags(&b->fork, cudaEventDisableTiming) != cudaSuccess) {
    b->fork = nullptr;
    return false;
  }
  for (int i = 0; i < kBatchSideStreams; ++i) {
    cudaStream_t st = nullptr;
    cudaEvent_t ev = nullptr;
    if (cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking) != cudaSuccess) break;
    if (cudaEventCreateWithFlags(&ev, cudaEventDisableTiming) != cudaSuccess) {
      cudaStreamDestroy(st);
      break;
    }
    b->side.push_back(st);
    b->join.push_back(ev);
  }
  if ((int)b->side.size() < kBatchSideStreams) {
    release_side_streams(b);
    cudaGetLastError();
    return false;
  }
  b->side_device = dev;
  return true;
}
constexpr int kBatchMaxOcc = 2048;
constexpr int64_t kBatchSumLimit = (int64_t)1 << 62;

struct BatchCarve {
  int64_t *weights, *inst_req, *req_off, *chunks, *tab_off, *opt, *F, *perm;
  uint32_t *split, *rows_scratch;
  int32_t *dfs, *status, *inst_list;
  uint8_t* flags;
};

size_t carve(const mpt_batch* b, char* base, BatchCarve* c) {
  size_t off = 0;
  auto take = [&](size_t bytes) -> char* {
    const size_t o = off;
    off += (bytes + 255) & ~(size_t)255;
    return base ? base + o : nullptr;
  };
  c->weights = reinterpret_cast<int64_t*>(take((size_t)b->n * 8));
  c->inst_req = reinterpret_cast<int64_t*>(take(((size_t)b->batch + 1) * 8));
  c->req_off = reinterpret_cast<int64_t*>(take(((size_t)b->requests + 1) * 8));
  c->chunks = reinterpret_cast<int64_t*>(take((size_t)std::max<int64_t>(b->occurrences, 1) * 8));
  c->tab_off = reinterpret_cast<int64_t*>(take(((size_t)b->batch + 1) * 8));
  c->opt = reinterpret_cast<int64_t*>(take((size_t)b->batch * 8));
  c->F = reinterpret_cast<int64_t*>(take((size_t)b->table_entries * 8));
  c->split = reinterpret_cast<uint32_t*>(take((size_t)b->table_entries * 4));
  c->perm = reinterpret_cast<int64_t*>(take((size_t)std::max<int64_t>(b->occurrences, 1) * 8));
  c->dfs = reinterpret_cast<int32_t*>(take((size_t)b->requests * 4));
  c->status = reinterpret_cast<int32_t*>(take((size_t)b->batch * 4));
  c->inst_list = reinterpret_cast<int32_t*>(take((size_t)b->batch * 4));
  c->flags = reinterpret_cast<uint8_t*>(take((size_t)b->batch));
  // rows of the row-blocked instances too large for shared memory, one slot
  // per block of their size's launch
  size_t scratch_words = 0;
  if (!b->group_rows_end.empty())
    for (int m = 1; m <= kBatchMaxM; ++m)
      scratch_words = std::max(scratch_words, (size_t)(b->group_rows_end[(size_t)m] - b->group_start[(size_t)m]) *
                                                  mpt::batch_rows_scratch_words(m));
  c->rows_scratch = scratch_words ? reinterpret_cast<uint32_t*>(take(scratch_words * 4)) : nullptr;
  return off;
}

}  // namespace

extern "C" {

mpt_status mpt_batch_create(const int64_t* weights, int64_t n_chunks, int32_t batch, const int64_t* inst_requests,
                            const int64_t* req_offsets, const int64_t* chunk_ids, mpt_batch** out) {
  if (!weights || !inst_requests || !req_offsets || !out || n_chunks < 1 || n_chunks > INT32_MAX || batch < 1)
    return MPT_ERR_INVALID_ARG;
  if (inst_requests[0] != 0) return MPT_ERR_INVALID_ARG;
  for (int32_t b = 0; b < batch; ++b) {
    const int64_t m = inst_requests[b + 1] - inst_requests[b];
    if (m < 1) return MPT_ERR_INVALID_ARG;
    if (m > kBatchMaxM) return MPT_ERR_TOO_LARGE;
  }
  const int64_t R = inst_requests[batch];
  if (req_offsets[0] != 0) return MPT_ERR_INVALID_ARG;
  for (int64_t r = 0; r < R; ++r)
    if (req_offsets[r + 1] < req_offsets[r]) return MPT_ERR_INVALID_ARG;
  const int64_t occ_total = req_offsets[R];
  if (occ_total > 0 && !chunk_ids) return MPT_ERR_INVALID_ARG;
  for (int64_t x = 0; x < n_chunks; ++x)
    if (weights[x] <= 0) return MPT_ERR_INVALID_ARG;
  mpt_batch* c = new (std::nothrow) mpt_batch();
  if (!c) return MPT_ERR_OUT_OF_MEMORY;
  try {
    c->tab_off.resize((size_t)batch + 1);
    c->flags.assign((size_t)batch, 0);
    std::vector<int> inst_occ((size_t)batch);
    int64_t tab = 0;
    std::vector<int64_t> ids;
    for (int32_t b = 0; b < batch; ++b) {
      const int64_t r0 = inst_requests[b], r1 = inst_requests[b + 1];
      const int m = (int)(r1 - r0);
      const int64_t occ = req_offsets[r1] - req_offsets[r0];
      if (occ > kBatchMaxOcc) {
        delete c;
        return MPT_ERR_TOO_LARGE;
      }
      for (int64_t r = r0; r < r1; ++r) {
        ids.assign(chunk_ids + req_offsets[r], chunk_ids + req_offsets[r + 1]);
        std::sort(ids.begin(), ids.end());
        for (size_t j = 0; j < ids.size(); ++j) {
          if (ids[j] < 0 || ids[j] >= n_chunks || (j > 0 && ids[j] == ids[j - 1])) {
            delete c;
            return MPT_ERR_INVALID_ARG;
          }
        }
      }
      // sum_i w(R_i) (below 2^62) and the shared weight W (below 2^31): the
      // request weight less the chunks that one or all m >= 2 requests hold,
      // which the kernels keep out of their 32-bit values (k_batch.cu)
      ids.assign(chunk_ids + req_offsets[r0], chunk_ids + req_offsets[r1]);
      std::sort(ids.begin(), ids.end());
      int64_t sum = 0, shared = 0;
      for (size_t j = 0; j < ids.size();) {
        size_t k = j;
        while (k < ids.size() && ids[k] == ids[j]) ++k;
        const int64_t cnt = (int64_t)(k - j), wx = weights[ids[j]];
        if (wx > (kBatchSumLimit - 1 - sum) / cnt) {
          delete c;
          return MPT_ERR_OVERFLOW;
        }
        sum += cnt * wx;
        if (cnt >= 2 && cnt < m) {
          shared += cnt * wx;
          if (shared >= ((int64_t)1 << 31)) {
            delete c;
            return MPT_ERR_OVERFLOW;
          }
        }
        j = k;
      }
      c->flags[(size_t)b] = (uint8_t)((shared < ((int64_t)1 << (32 - m)) ? mpt::kFlagPacked : 0) |
                                      (sum >= ((int64_t)1 << (32 - m)) ? mpt::kFlagOffsets : 0));
      // the instance's kernel must hold its shared-memory arrays: the
      // per-subset kernel keeps the 2^m tables there (m = 15: room for 1024
      // occurrences; m = 16 does not fit, so 16 requests need packed keys),
      // the row-blocked kernel its rows up to m = 15
      int cap = 1;
      while (cap < occ) cap <<= 1;
      const bool rows = m >= 6 && (c->flags[(size_t)b] & mpt::kFlagPacked);
      if ((rows ? mpt::batch_rows_smem_bytes(m, cap) : mpt::batch_smem_bytes(m, cap)) > kBatchMaxSmem) {
        delete c;
        return MPT_ERR_TOO_LARGE;
      }
      c->tab_off[(size_t)b] = tab;
      tab += (int64_t)1 << m;
      c->max_m = std::max(c->max_m, m);
      while (c->occ_cap < occ) c->occ_cap <<= 1;
      inst_occ[(size_t)b] = (int)occ;
    }
    c->tab_off[(size_t)batch] = tab;
    // group the instances by m (stable), each group with its own occurrence cap
    c->group_start.assign(kBatchMaxM + 2, 0);
    for (int32_t b = 0; b < batch; ++b) ++c->group_start[(size_t)(inst_requests[b + 1] - inst_requests[b]) + 1];
    for (int m = 1; m <= kBatchMaxM + 1; ++m) c->group_start[(size_t)m] += c->group_start[(size_t)m - 1];
    c->inst_list.resize((size_t)batch);
    c->group_occ_cap_rows.assign(kBatchMaxM + 1, 1);
    c->group_occ_cap.assign(kBatchMaxM + 1, 1);
    std::vector<int64_t> fill(c->group_start.begin(), c->group_start.end());
    for (int pass = 0; pass < 2; ++pass) {
      for (int32_t b = 0; b < batch; ++b) {
        const int m = (int)(inst_requests[b + 1] - inst_requests[b]);
        const bool rows = m >= 6 && (c->flags[(size_t)b] & mpt::kFlagPacked);
        if (rows != (pass == 0)) continue;
        c->inst_list[(size_t)fill[(size_t)m]++] = b;
        int& cap = rows ? c->group_occ_cap_rows[(size_t)m] : c->group_occ_cap[(size_t)m];
        while (cap < inst_occ[(size_t)b]) cap <<= 1;
      }
      if (pass == 0) c->group_rows_end.assign(fill.begin(), fill.end());
    }
    c->table_entries = tab;
    c->w.assign(weights, weights + n_chunks);
    c->inst_req.assign(inst_requests, inst_requests + batch + 1);
    c->req_off.assign(req_offsets, req_offsets + R + 1);
    if (occ_total) c->chunks.assign(chunk_ids, chunk_ids + occ_total);
  } catch (...) {
    delete c;
    return MPT_ERR_OUT_OF_MEMORY;
  }
  c->batch = batch;
  c->n = n_chunks;
  c->requests = R;
  c->occurrences = occ_total;
  *out = c;
  return MPT_OK;
}

mpt_status mpt_batch_workspace_bytes(const mpt_batch* b, size_t* bytes) {
  if (!b || !bytes) return MPT_ERR_INVALID_ARG;
  BatchCarve c{};
  *bytes = carve(b, nullptr, &c);
  return MPT_OK;
}

mpt_status mpt_batch_solve(mpt_batch* b, void* d_workspace, size_t workspace_bytes, void* stream_ptr) {
  if (!b) return MPT_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_ptr);
  b->solved = false;
  BatchCarve c{};
  const size_t need = carve(b, nullptr, &c);
  char* base = nullptr;
  if (d_workspace) {
    if (workspace_bytes < need) return MPT_ERR_WORKSPACE_TOO_SMALL;
    if (reinterpret_cast<uintptr_t>(d_workspace) & 255) return MPT_ERR_INVALID_ARG;
    base = static_cast<char*>(d_workspace);
  } else {
    if (b->own_bytes < need) {
      if (b->own_ws) cudaFree(b->own_ws);
      b->own_ws = nullptr;
      b->own_bytes = 0;
      if (mpt::device_alloc(&b->own_ws, need) != cudaSuccess) return MPT_ERR_OUT_OF_MEMORY;
      b->own_bytes = need;
    }
    base = static_cast<char*>(b->own_ws);
  }
  carve(b, base, &c);
  const size_t B = (size_t)b->batch;
  try {
    b->opt.resize(B);
    b->status.resize(B);
    b->perm.resize((size_t)b->occurrences);
    b->dfs.resize((size_t)b->requests);
  } catch (...) {
    return MPT_ERR_OUT_OF_MEMORY;
  }
  cudaError_t e = cudaSuccess;
  auto h2d = [&](void* d, const void* h, size_t bytes) {
    if (e == cudaSuccess && bytes) e = cudaMemcpyAsync(d, h, bytes, cudaMemcpyHostToDevice, stream);
  };
  auto d2h = [&](void* h, const void* d, size_t bytes) {
    if (e == cudaSuccess && bytes) e = cudaMemcpyAsync(h, d, bytes, cudaMemcpyDeviceToHost, stream);
  };
  h2d(c.weights, b->w.data(), (size_t)b->n * 8);
  h2d(c.inst_req, b->inst_req.data(), (B + 1) * 8);
  h2d(c.req_off, b->req_off.data(), ((size_t)b->requests + 1) * 8);
  h2d(c.chunks, b->chunks.data(), (size_t)b->occurrences * 8);
  h2d(c.tab_off, b->tab_off.data(), (B + 1) * 8);
  h2d(c.inst_list, b->inst_list.data(), B * 4);
  h2d(c.flags, b->flags.data(), B);
  // One grid per instance size, largest first.  The grids write disjoint
  // instances, so they run on side streams forked from the caller's stream
  // after the uploads and joined back before the downloads: the short grids
  // of small sizes then fill the SMs that the long ones leave idle.
  const bool forked = e == cudaSuccess && side_streams(b);
  if (forked) {
    e = cudaEventRecord(b->fork, stream);
    for (int i = 0; i < kBatchSideStreams && e == cudaSuccess; ++i) e = cudaStreamWaitEvent(b->side[(size_t)i], b->fork, 0);
  }
  int next_side = 0;
  for (int m = kBatchMaxM; m >= 1 && e == cudaSuccess; --m) {
    const int64_t g0 = b->group_start[(size_t)m], gr = b->group_rows_end[(size_t)m],
                  g1 = b->group_start[(size_t)m + 1];
    if (g1 == g0) continue;
    cudaStream_t st = forked ? b->side[(size_t)(next_side++ % kBatchSideStreams)] : stream;
    if (gr > g0)
      e = mpt::launch_batch_rows((int)(gr - g0), m, b->group_occ_cap_rows[(size_t)m], c.weights, c.inst_req, c.req_off,
                                 c.chunks, c.tab_off, c.inst_list + g0, c.flags, c.opt, c.F, c.split, c.perm, c.dfs,
                                 c.status, c.rows_scratch, st);
    if (e == cudaSuccess && g1 > gr)
      e = mpt::launch_batch((int)(g1 - gr), m, b->group_occ_cap[(size_t)m], c.weights, c.inst_req, c.req_off,
                            c.chunks, c.tab_off, c.inst_list + gr, c.flags, c.opt, c.F, c.split, c.perm, c.dfs,
                            c.status, st);
  }
  if (forked) {
    // join every side stream, also after a failed launch, so that no work
    // of this call runs on after it returns
    for (int i = 0; i < kBatchSideStreams; ++i) {
      cudaError_t ej = cudaEventRecord(b->join[(size_t)i], b->side[(size_t)i]);
      if (ej == cudaSuccess) ej = cudaStreamWaitEvent(stream, b->join[(size_t)i], 0);
      if (ej != cudaSuccess) {
        cudaStreamSynchronize(b->side[(size_t)i]);
        if (e == cudaSuccess) e = ej;
      }
    }
  }
  d2h(b->opt.data(), c.opt, B * 8);
  d2h(b->status.data(), c.status, B * 4);
  d2h(b->perm.data(), c.perm, (size_t)b->occurrences * 8);
  d2h(b->dfs.data(), c.dfs, (size_t)b->requests * 4);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e == cudaErrorMemoryAllocation ? MPT_ERR_OUT_OF_MEMORY : MPT_ERR_CUDA;
  for (size_t i = 0; i < B; ++i)
    if (b->status[i] != 0) return MPT_ERR_INTERNAL;
  b->d_F = c.F;
  b->d_split = c.split;
  b->solved = true;
  return MPT_OK;
}

mpt_status mpt_batch_results(const mpt_batch* b, int64_t* opt, int64_t* perm_chunks, int32_t* dfs_order) {
  if (!b) return MPT_ERR_INVALID_ARG;
  if (!b->solved) return MPT_ERR_NOT_SOLVED;
  if (opt) std::memcpy(opt, b->opt.data(), b->opt.size() * 8);
  if (perm_chunks && !b->perm.empty()) std::memcpy(perm_chunks, b->perm.data(), b->perm.size() * 8);
  if (dfs_order && !b->dfs.empty()) std::memcpy(dfs_order, b->dfs.data(), b->dfs.size() * 4);
  return MPT_OK;
}

mpt_status mpt_batch_tables(const mpt_batch* b, const int64_t** d_F, const uint32_t** d_split,
                            int64_t* table_offsets) {
  if (!b) return MPT_ERR_INVALID_ARG;
  if (!b->solved) return MPT_ERR_NOT_SOLVED;
  if (d_F) *d_F = b->d_F;
  if (d_split) *d_split = b->d_split;
  if (table_offsets) std::memcpy(table_offsets, b->tab_off.data(), b->tab_off.size() * 8);
  return MPT_OK;
}

void mpt_batch_destroy(mpt_batch* b) {
  if (!b) return;
  if (b->own_ws) cudaFree(b->own_ws);
  release_side_streams(b);
  delete b;
}

}  // extern "C"
