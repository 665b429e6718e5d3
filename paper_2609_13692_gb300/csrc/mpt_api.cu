// C ABI of the exact MPT solver (include/mpt.h): argument checks, workspace
// carve-up and the order of launches.  Every step of the solve itself runs in
// the kernels of k_scatter_zeta.cu, k_dp_blocked.cu / k_dp_general.cu and
// k_walk.cu, all on the caller's stream.
#include <climits>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "../../include/mpt.h"
#include "mpt_internal.cuh"

struct mpt_ctx {
  mpt::Shape shape{};
  std::vector<int64_t> w;
  std::vector<uint64_t> bits;
  int64_t sum_w = 0;     // sum_i w(R_i)
  int64_t shared_w = 0;  // the same less the chunks one or every request needs
  int32_t mode = MPT_DP_AUTO;
  int32_t tables = MPT_TABLES_INT64;
  void* own_ws = nullptr;
  size_t own_bytes = 0;
  bool solved = false;
  int64_t opt = 0;
  std::vector<int64_t> h_offsets, h_chunks;
  std::vector<int32_t> h_dfs;
  std::string err;
  bool profiling = false;
  mpt_profile prof{};
  std::vector<cudaEvent_t> events;
  mpt::Workspace ws{};  // carve-up of the last successful solve
  char* resident = nullptr;  // workspace whose input copies hold this context's instance
  int32_t staged_next = -1;  // staged solve: next step of the recurrence (-1: none begun)
  char* staged_base = nullptr;  // staged solve: its workspace
  // blocked solves leave the tables in rotated order; the natural views are
  // filled on the first mpt_tables / mpt_tables32 call after the solve, on a
  // stream of the context, on the device of the solve
  bool natural = false;
  int device = 0;
  cudaStream_t conv_stream = nullptr;
  int conv_device = -1;
};

namespace {

constexpr int kMaxRequests = 32;
constexpr int64_t kSumLimit = (int64_t)1 << 62;

constexpr int64_t kWideLimit = (int64_t)1 << 51;  // 64-bit keys: F(A) + F(B) < 2^52

// The blocked recurrence runs on F' = F - pi(S) (k_scatter_zeta.cu), whose
// candidates F'(A) + F'(B) stay at most the shared weight.
bool blocked_feasible(const mpt_ctx* c) {
  const int b = mpt::blocked_tile_bits(c->shape.m);
  return c->shared_w < ((int64_t)1 << (32 - b));
}

bool wide_feasible(const mpt_ctx* c) { return c->shared_w < kWideLimit; }

bool use_blocked(const mpt_ctx* c) {
  if (c->mode == MPT_DP_GENERAL) return false;
  if (c->mode == MPT_DP_BLOCKED) return blocked_feasible(c);
  return wide_feasible(c);  // AUTO and WIDE: the 32- or the 64-bit keys
}

bool use_wide(const mpt_ctx* c) {
  if (c->mode == MPT_DP_WIDE) return wide_feasible(c);
  return c->mode == MPT_DP_AUTO && !blocked_feasible(c) && wide_feasible(c);
}

void refresh_shape(mpt_ctx* c) {
  mpt::Shape& s = c->shape;
  s.blocked = use_blocked(c);
  s.wide = s.blocked && use_wide(c);
  s.lean = c->tables == MPT_TABLES_LEAN;
  s.b = mpt::blocked_tile_bits(s.m);
  s.L = s.m - s.b;
  s.partial_entries = !s.blocked ? 0
                      : s.wide   ? (mpt::wide_partial_slots(s.m, s.b) << s.b)
                                 : mpt::blocked_partial_entries(s.m, s.b);
}

mpt_status cuda_fail(mpt_ctx* c, cudaError_t e, const char* what) {
  char buf[256];
  std::snprintf(buf, sizeof(buf), "%s: %s", what, cudaGetErrorString(e));
  c->err = buf;
  return e == cudaErrorMemoryAllocation ? MPT_ERR_OUT_OF_MEMORY : MPT_ERR_CUDA;
}

#define MPT_CK(call, what)                      \
  do {                                          \
    cudaError_t e_ = (call);                    \
    if (e_ != cudaSuccess) return cuda_fail(c, e_, what); \
  } while (0)

}  // namespace

namespace mpt {

size_t carve_workspace(const Shape& s, char* base, Workspace* ws) {
  size_t off = 0;
  auto take = [&](size_t bytes) -> char* {
    const size_t o = off;
    off += (bytes + 255) & ~(size_t)255;
    return base ? base + o : nullptr;
  };
  const size_t N = (size_t)1 << s.m;
  const size_t slots = s.slots > 0 ? (size_t)s.slots : 1;
  ws->weights = reinterpret_cast<int64_t*>(take((size_t)s.n * 8));
  ws->bits = reinterpret_cast<uint64_t*>(take((size_t)s.m * (size_t)s.words * 8));
  ws->used_N = reinterpret_cast<uint32_t*>(take(slots * 4));
  ws->used_x = reinterpret_cast<int32_t*>(take(slots * 4));
  ws->counters = reinterpret_cast<int32_t*>(take(8 * 4));
  if (s.lean) {
    ws->fw = reinterpret_cast<int32_t*>(take(N * 4));
    ws->wI = ws->F = nullptr;
  } else {
    ws->wI = reinterpret_cast<int64_t*>(take(N * 8));
    ws->F = reinterpret_cast<int64_t*>(take(N * 8));
    ws->fw = nullptr;
  }
  ws->split = reinterpret_cast<uint32_t*>(take(N * 4));
  ws->Gp64 = ws->Gc64 = nullptr;
  ws->partial_ta = nullptr;
  if (s.blocked && s.wide) {
    ws->Gp64 = reinterpret_cast<unsigned long long*>(take(N * 8));
    ws->Gc64 = reinterpret_cast<unsigned long long*>(take(N * 8));
    ws->Gp = ws->Gc = nullptr;
    const size_t pe = (size_t)(s.partial_entries > 0 ? s.partial_entries : 1);
    ws->partial = reinterpret_cast<unsigned long long*>(take(pe * 8));
    ws->partial_ta = reinterpret_cast<uint32_t*>(take(pe * 4));
  } else if (s.blocked) {
    ws->Gp = reinterpret_cast<uint32_t*>(take(N * 4));
    ws->Gc = reinterpret_cast<uint32_t*>(take(N * 4));
    ws->partial = reinterpret_cast<unsigned long long*>(take((size_t)(s.partial_entries > 0 ? s.partial_entries : 1) * 8));
  }
  ws->priv = s.blocked ? reinterpret_cast<unsigned long long*>(take(mpt::kOffsetSlots * 8)) : nullptr;
  if (s.blocked) {
    // The rotated tables share the buffers of the natural ones: w(I) sits in
    // the F table (int64) or in fw (lean), split in the split table.  The
    // natural views, when asked for, go to wI, F or fw (F from Gp) and, for
    // split, to the Gc table (32- or 64-bit), which the recurrence no longer
    // needs.
    ws->wI_rot = s.lean ? nullptr : ws->F;
    ws->fw_rot = s.lean ? ws->fw : nullptr;
    ws->split_rot = ws->split;
  } else {
    ws->Gp = ws->Gc = nullptr;
    ws->partial = nullptr;
    ws->wI_rot = nullptr;
    ws->fw_rot = nullptr;
    ws->split_rot = nullptr;
  }
  ws->keys = reinterpret_cast<unsigned long long*>(take(slots * 8));
  ws->perm_offsets = reinterpret_cast<int64_t*>(take((size_t)(s.m + 1) * 8));
  ws->perm_chunks = reinterpret_cast<int64_t*>(take(slots * 8));
  ws->dfs = reinterpret_cast<int32_t*>(take((size_t)s.m * 4));
  ws->opt = reinterpret_cast<int64_t*>(take(8));
  return off;
}

}  // namespace mpt

extern "C" {

const char* mpt_status_string(mpt_status s) {
  switch (s) {
    case MPT_OK: return "ok";
    case MPT_ERR_INVALID_ARG: return "invalid argument";
    case MPT_ERR_TOO_LARGE: return "instance beyond the documented limits";
    case MPT_ERR_OVERFLOW: return "weights too large for the requested arithmetic";
    case MPT_ERR_OUT_OF_MEMORY: return "out of memory";
    case MPT_ERR_WORKSPACE_TOO_SMALL: return "workspace too small";
    case MPT_ERR_CUDA: return "CUDA error";
    case MPT_ERR_NOT_SOLVED: return "no successful solve yet";
    case MPT_ERR_TIMEOUT: return "device wait timed out";
    case MPT_ERR_INTERNAL: return "internal consistency check failed";
  }
  return "unknown status";
}

const char* mpt_last_error(const mpt_ctx* ctx) { return ctx ? ctx->err.c_str() : ""; }

mpt_status mpt_build_info(int32_t* flags) {
  if (!flags) return MPT_ERR_INVALID_ARG;
  *flags = mpt::kBoundsChecked ? 1 : 0;
  return MPT_OK;
}

mpt_status mpt_create(const int64_t* weights, int64_t n_chunks, const uint64_t* req_bits, int32_t m, mpt_ctx** out) {
  if (!weights || !req_bits || !out || n_chunks < 1 || n_chunks > INT32_MAX || m < 1) return MPT_ERR_INVALID_ARG;
  if (m > kMaxRequests) return MPT_ERR_TOO_LARGE;
  const int64_t words = (n_chunks + 63) / 64;
  for (int64_t x = 0; x < n_chunks; ++x)
    if (weights[x] <= 0) return MPT_ERR_INVALID_ARG;
  const int tail = (int)(n_chunks & 63);
  int64_t slots = 0;
  int64_t sum = 0;
  for (int i = 0; i < m; ++i) {
    const uint64_t* row = req_bits + (size_t)i * (size_t)words;
    if (tail && (row[words - 1] >> tail) != 0) return MPT_ERR_INVALID_ARG;
    for (int64_t j = 0; j < words; ++j) {
      for (uint64_t v = row[j]; v; v &= v - 1) {
        const int64_t x = j * 64 + __builtin_ctzll(v);
        ++slots;
        if (sum > kSumLimit - weights[x]) return MPT_ERR_OVERFLOW;
        sum += weights[x];
      }
    }
  }
  // request weight the packed keys leave out (k_scatter_zeta.cu): the chunks
  // exactly one request needs (per word, the bits seen once, s1, but not
  // twice, s2) and, for m >= 2, m times those that every request needs
  int64_t private_w = 0;
  for (int64_t j = 0; j < words; ++j) {
    uint64_t s1 = 0, s2 = 0, all = ~0ull;
    for (int i = 0; i < m; ++i) {
      const uint64_t v = req_bits[(size_t)i * (size_t)words + (size_t)j];
      s2 |= s1 & v;
      s1 |= v;
      all &= v;
    }
    for (uint64_t v = s1 & ~s2; v; v &= v - 1) private_w += weights[j * 64 + __builtin_ctzll(v)];
    if (m >= 2)
      for (uint64_t v = all; v; v &= v - 1) private_w += (int64_t)m * weights[j * 64 + __builtin_ctzll(v)];
  }
  mpt_ctx* c = new (std::nothrow) mpt_ctx();
  if (!c) return MPT_ERR_OUT_OF_MEMORY;
  try {
    c->w.assign(weights, weights + n_chunks);
    c->bits.assign(req_bits, req_bits + (size_t)m * (size_t)words);
  } catch (...) {
    delete c;
    return MPT_ERR_OUT_OF_MEMORY;
  }
  c->shape.m = m;
  c->shape.n = n_chunks;
  c->shape.words = words;
  c->shape.slots = slots;
  c->sum_w = sum;
  c->shared_w = sum - private_w;
  refresh_shape(c);
  *out = c;
  return MPT_OK;
}

mpt_status mpt_workspace_bytes(const mpt_ctx* ctx, size_t* bytes) {
  if (!ctx || !bytes) return MPT_ERR_INVALID_ARG;
  mpt::Workspace ws{};
  *bytes = mpt::carve_workspace(ctx->shape, nullptr, &ws);
  return MPT_OK;
}

mpt_status mpt_set_dp_mode(mpt_ctx* ctx, int32_t mode) {
  if (!ctx || mode < MPT_DP_AUTO || mode > MPT_DP_WIDE) return MPT_ERR_INVALID_ARG;
  if (mode == MPT_DP_BLOCKED && !blocked_feasible(ctx)) return MPT_ERR_OVERFLOW;
  if (mode == MPT_DP_WIDE && !wide_feasible(ctx)) return MPT_ERR_OVERFLOW;
  ctx->mode = mode;
  refresh_shape(ctx);
  ctx->solved = false;
  ctx->staged_next = -1;
  ctx->resident = nullptr;  // the carve-up may move the input copies
  return MPT_OK;
}

mpt_status mpt_set_tables(mpt_ctx* ctx, int32_t kind) {
  if (!ctx || (kind != MPT_TABLES_INT64 && kind != MPT_TABLES_LEAN)) return MPT_ERR_INVALID_ARG;
  if (kind == MPT_TABLES_LEAN && ctx->sum_w >= ((int64_t)1 << 31)) return MPT_ERR_OVERFLOW;
  ctx->tables = kind;
  refresh_shape(ctx);
  ctx->solved = false;
  ctx->staged_next = -1;
  ctx->resident = nullptr;  // the carve-up moves
  return MPT_OK;
}

mpt_status mpt_set_profiling(mpt_ctx* ctx, int32_t on) {
  if (!ctx) return MPT_ERR_INVALID_ARG;
  ctx->profiling = on != 0;
  return MPT_OK;
}

mpt_status mpt_get_profile(const mpt_ctx* ctx, mpt_profile* out) {
  if (!ctx || !out) return MPT_ERR_INVALID_ARG;
  if (!ctx->solved) return MPT_ERR_NOT_SOLVED;
  *out = ctx->prof;
  return MPT_OK;
}

static float elapsed(cudaEvent_t a, cudaEvent_t b) {
  float ms = 0.f;
  cudaEventElapsedTime(&ms, a, b);
  return ms;
}

namespace {

// Resolve the workspace of a solve (the caller's, or one the context owns)
// and carve it.
mpt_status bind_workspace(mpt_ctx* c, void* d_workspace, size_t workspace_bytes, mpt::Workspace* ws, char** base) {
  const mpt::Shape& s = c->shape;
  const size_t need = mpt::carve_workspace(s, nullptr, ws);
  if (d_workspace) {
    if (workspace_bytes < need) return MPT_ERR_WORKSPACE_TOO_SMALL;
    if (reinterpret_cast<uintptr_t>(d_workspace) & 255) return MPT_ERR_INVALID_ARG;
    *base = static_cast<char*>(d_workspace);
  } else {
    if (c->own_bytes < need) {
      if (c->own_ws) cudaFree(c->own_ws);
      c->own_ws = nullptr;
      c->own_bytes = 0;
      c->resident = nullptr;
      MPT_CK(mpt::device_alloc(&c->own_ws, need), "cudaMalloc(workspace)");
      c->own_bytes = need;
    }
    *base = static_cast<char*>(c->own_ws);
  }
  mpt::carve_workspace(s, *base, ws);
  return MPT_OK;
}

// Input copies (unless this workspace already holds them), K1 and K2.
mpt_status run_front(mpt_ctx* c, const mpt::Workspace& ws, char* base, cudaStream_t stream, int* launches,
                     cudaEvent_t* ev) {
  const mpt::Shape& s = c->shape;
  auto mark = [&](int i) {
    if (ev) cudaEventRecord(ev[i], stream);
  };
  const size_t N = (size_t)1 << s.m;
  mark(0);
  if (c->resident != base) {
    c->resident = nullptr;
    MPT_CK(cudaMemcpyAsync(ws.weights, c->w.data(), (size_t)s.n * 8, cudaMemcpyHostToDevice, stream), "copy weights");
    MPT_CK(cudaMemcpyAsync(ws.bits, c->bits.data(), c->bits.size() * 8, cudaMemcpyHostToDevice, stream), "copy bits");
  }
  MPT_CK(cudaMemsetAsync(ws.counters, 0, 8 * 4, stream), "memset counters");
  if (ws.priv) MPT_CK(cudaMemsetAsync(ws.priv, 0, mpt::kOffsetSlots * 8, stream), "memset offsets");
  MPT_CK(cudaMemsetAsync(mpt::g_table(s, ws), 0, N * (s.lean ? 4 : 8), stream), "memset g");
  mark(1);
  MPT_CK(mpt::launch_scatter(s, ws, stream, launches), "scatter kernel");
  mark(2);
  MPT_CK(mpt::launch_zeta(s, ws, stream, launches), "zeta kernels");
  mark(3);
  return MPT_OK;
}

// Steps [begin, end) of the recurrence.
mpt_status run_steps(mpt_ctx* c, const mpt::Workspace& ws, cudaStream_t stream, int* launches,
                     mpt::BlockedTiming* timing, int begin, int end) {
  const mpt::Shape& s = c->shape;
  if (s.blocked && s.wide) {
    MPT_CK(mpt::launch_dp_wide(s, ws, stream, launches, timing, begin, end), "wide blocked DP kernels");
  } else if (s.blocked) {
    MPT_CK(mpt::launch_dp_blocked(s, ws, stream, launches, timing, begin, end), "blocked DP kernels");
  } else {
    MPT_CK(mpt::launch_dp_general(s, ws, stream, launches, begin, end), "general DP kernels");
  }
  return MPT_OK;
}

// The walk, the copies of its results and the consistency flags.
mpt_status run_back(mpt_ctx* c, const mpt::Workspace& ws, cudaStream_t stream, int* launches, cudaEvent_t* ev,
                    int64_t* opt_out) {
  const mpt::Shape& s = c->shape;
  auto mark = [&](int i) {
    if (ev) cudaEventRecord(ev[i], stream);
  };
  MPT_CK(mpt::launch_walk(s, ws, stream, launches), "walk kernel");
  mark(5);
  int32_t counters[8];
  int64_t opt = 0;
  const size_t slots = (size_t)s.slots;
  try {
    c->h_offsets.resize((size_t)s.m + 1);
    c->h_chunks.resize(slots);
    c->h_dfs.resize((size_t)s.m);
  } catch (...) {
    return MPT_ERR_OUT_OF_MEMORY;
  }
  MPT_CK(cudaMemcpyAsync(&opt, ws.opt, 8, cudaMemcpyDeviceToHost, stream), "copy opt");
  MPT_CK(cudaMemcpyAsync(counters, ws.counters, sizeof(counters), cudaMemcpyDeviceToHost, stream), "copy flags");
  MPT_CK(cudaMemcpyAsync(c->h_offsets.data(), ws.perm_offsets, ((size_t)s.m + 1) * 8, cudaMemcpyDeviceToHost, stream),
         "copy offsets");
  if (slots)
    MPT_CK(cudaMemcpyAsync(c->h_chunks.data(), ws.perm_chunks, slots * 8, cudaMemcpyDeviceToHost, stream),
           "copy chunks");
  MPT_CK(cudaMemcpyAsync(c->h_dfs.data(), ws.dfs, (size_t)s.m * 4, cudaMemcpyDeviceToHost, stream), "copy dfs");
  mark(6);
  MPT_CK(cudaStreamSynchronize(stream), "solve");
  if (counters[1] != 0) {
    char buf[128];
    std::snprintf(buf, sizeof(buf), "device consistency flags 0x%x", counters[1]);
    c->err = buf;
    return (counters[1] & mpt::kErrTimeout) ? MPT_ERR_TIMEOUT : MPT_ERR_INTERNAL;
  }
  *opt_out = opt;
  return MPT_OK;
}

}  // namespace

mpt_status mpt_solve(mpt_ctx* ctx, void* d_workspace, size_t workspace_bytes, void* stream_ptr, int64_t* opt_cost) {
  mpt_ctx* c = ctx;
  if (!c || !opt_cost) return MPT_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_ptr);
  const mpt::Shape& s = c->shape;
  c->solved = false;
  c->staged_next = -1;
  c->err.clear();

  mpt::Workspace ws{};
  char* base = nullptr;
  mpt_status st = bind_workspace(c, d_workspace, workspace_bytes, &ws, &base);
  if (st != MPT_OK) return st;

  // events: 7 stage marks + 2 per blocked-DP launch
  const int dp_launches = mpt::blocked_max_launches(s);
  const size_t n_events = 7 + 4 * (size_t)dp_launches;
  if (c->profiling && c->events.size() < n_events) {
    while (c->events.size() < n_events) {
      cudaEvent_t e;
      MPT_CK(cudaEventCreate(&e), "cudaEventCreate");
      c->events.push_back(e);
    }
  }
  cudaEvent_t* ev = c->profiling ? c->events.data() : nullptr;

  int launches = 0;
  const size_t N = (size_t)1 << s.m;
  if ((st = run_front(c, ws, base, stream, &launches, ev)) != MPT_OK) return st;
  mpt::BlockedTiming timing{};
  if (s.blocked) {
    timing.pair_ev = ev ? ev + 7 : nullptr;
    timing.tile_ev = ev ? ev + 7 + 2 * dp_launches : nullptr;
  }
  if ((st = run_steps(c, ws, stream, &launches, &timing, 0, -1)) != MPT_OK) return st;
  if (ev) cudaEventRecord(ev[4], stream);
  int64_t opt = 0;
  if ((st = run_back(c, ws, stream, &launches, ev, &opt)) != MPT_OK) return st;
  c->ws = ws;
  c->opt = opt;
  c->resident = base;

  mpt_profile& p = c->prof;
  std::memset(&p, 0, sizeof(p));
  p.launches_total = launches;
  p.dp_mode = !s.blocked ? MPT_DP_GENERAL : (s.wide ? MPT_DP_WIDE : MPT_DP_BLOCKED);
  p.tile_bits = s.blocked ? s.b : 0;
  {
    // (3^m + 1)/2 - 2^m, exactly representable in a double for m <= 32
    double three = 1.0;
    for (int i = 0; i < s.m; ++i) three *= 3.0;
    p.splits_total = (three + 1.0) / 2.0 - (double)N;
  }
  p.splits_pairs = timing.pair_splits;
  p.launches_pairs = timing.pair_launches;
  if (ev) {
    p.ms_h2d = elapsed(ev[0], ev[1]);
    p.ms_scatter = elapsed(ev[1], ev[2]);
    p.ms_zeta = elapsed(ev[2], ev[3]);
    if (s.blocked) {
      for (int i = 0; i < timing.pair_launches; ++i) p.ms_dp_pairs += elapsed(timing.pair_ev[2 * i], timing.pair_ev[2 * i + 1]);
      for (int i = 0; i < timing.tile_launches; ++i) p.ms_dp_tiles += elapsed(timing.tile_ev[2 * i], timing.tile_ev[2 * i + 1]);
    } else {
      p.ms_dp_general = elapsed(ev[3], ev[4]);
    }
    p.ms_walk = elapsed(ev[4], ev[5]);
    p.ms_d2h = elapsed(ev[5], ev[6]);
  }
  c->natural = !s.blocked;
  cudaGetDevice(&c->device);
  c->solved = true;
  *opt_cost = opt;
  return MPT_OK;
}

mpt_status mpt_solve_steps(const mpt_ctx* ctx, int32_t* steps) {
  if (!ctx || !steps) return MPT_ERR_INVALID_ARG;
  *steps = mpt::dp_steps(ctx->shape);
  return MPT_OK;
}

mpt_status mpt_solve_begin(mpt_ctx* ctx, void* d_workspace, size_t workspace_bytes, void* stream_ptr) {
  mpt_ctx* c = ctx;
  if (!c) return MPT_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_ptr);
  c->solved = false;
  c->staged_next = -1;
  c->err.clear();
  mpt::Workspace ws{};
  char* base = nullptr;
  mpt_status st = bind_workspace(c, d_workspace, workspace_bytes, &ws, &base);
  if (st != MPT_OK) return st;
  int launches = 0;
  if ((st = run_front(c, ws, base, stream, &launches, nullptr)) != MPT_OK) return st;
  if ((st = run_steps(c, ws, stream, &launches, nullptr, 0, 1)) != MPT_OK) return st;
  c->resident = base;
  c->staged_base = base;
  c->staged_next = 1;
  return MPT_OK;
}

mpt_status mpt_solve_resume(mpt_ctx* ctx, void* d_workspace, size_t workspace_bytes, int32_t next_step) {
  mpt_ctx* c = ctx;
  if (!c || !d_workspace) return MPT_ERR_INVALID_ARG;
  if (next_step < 1 || next_step > mpt::dp_steps(c->shape)) return MPT_ERR_INVALID_ARG;
  mpt::Workspace ws{};
  char* base = nullptr;
  mpt_status st = bind_workspace(c, d_workspace, workspace_bytes, &ws, &base);
  if (st != MPT_OK) return st;
  c->solved = false;
  c->resident = base;  // a checkpoint carries the input copies with it
  c->staged_base = base;
  c->staged_next = next_step;
  return MPT_OK;
}

mpt_status mpt_solve_layers(mpt_ctx* ctx, void* d_workspace, size_t workspace_bytes, void* stream_ptr, int32_t count,
                            int32_t* next_step) {
  mpt_ctx* c = ctx;
  if (!c || count < 0) return MPT_ERR_INVALID_ARG;
  if (c->staged_next < 0) return MPT_ERR_NOT_SOLVED;
  mpt::Workspace ws{};
  char* base = nullptr;
  mpt_status st = bind_workspace(c, d_workspace, workspace_bytes, &ws, &base);
  if (st != MPT_OK) return st;
  if (base != c->staged_base) return MPT_ERR_INVALID_ARG;
  const int total = mpt::dp_steps(c->shape);
  const int end = c->staged_next + count < total ? c->staged_next + count : total;
  int launches = 0;
  if ((st = run_steps(c, ws, reinterpret_cast<cudaStream_t>(stream_ptr), &launches, nullptr, c->staged_next, end)) !=
      MPT_OK)
    return st;
  c->staged_next = end;
  if (next_step) *next_step = end;
  return MPT_OK;
}

mpt_status mpt_solve_end(mpt_ctx* ctx, void* d_workspace, size_t workspace_bytes, void* stream_ptr, int64_t* opt_cost) {
  mpt_ctx* c = ctx;
  if (!c || !opt_cost) return MPT_ERR_INVALID_ARG;
  if (c->staged_next < 0 || c->staged_next != mpt::dp_steps(c->shape)) return MPT_ERR_NOT_SOLVED;
  mpt::Workspace ws{};
  char* base = nullptr;
  mpt_status st = bind_workspace(c, d_workspace, workspace_bytes, &ws, &base);
  if (st != MPT_OK) return st;
  if (base != c->staged_base) return MPT_ERR_INVALID_ARG;
  int launches = 0;
  int64_t opt = 0;
  if ((st = run_back(c, ws, reinterpret_cast<cudaStream_t>(stream_ptr), &launches, nullptr, &opt)) != MPT_OK) return st;
  c->ws = ws;
  c->opt = opt;
  c->staged_next = -1;
  std::memset(&c->prof, 0, sizeof(c->prof));
  c->natural = !c->shape.blocked;
  cudaGetDevice(&c->device);
  c->solved = true;
  *opt_cost = opt;
  return MPT_OK;
}

}  // extern "C"

namespace {

// Fill the natural-order views of a blocked solve's tables (once per solve).
mpt_status ensure_natural(mpt_ctx* c) {
  if (c->natural) return MPT_OK;
  const mpt::Shape& s = c->shape;
  const mpt::Workspace& ws = c->ws;
  int prev = 0;
  MPT_CK(cudaGetDevice(&prev), "cudaGetDevice");
  MPT_CK(cudaSetDevice(c->device), "cudaSetDevice");
  mpt_status st = MPT_OK;
  cudaError_t e = cudaSuccess;
  if (c->conv_stream && c->conv_device != c->device) {
    cudaStreamDestroy(c->conv_stream);
    c->conv_stream = nullptr;
  }
  if (!c->conv_stream) {
    e = cudaStreamCreateWithFlags(&c->conv_stream, cudaStreamNonBlocking);
    c->conv_device = c->device;
  }
  if (e == cudaSuccess && s.wide)
    e = mpt::unrotate_tables_wide(s, ws.split_rot, reinterpret_cast<uint32_t*>(ws.Gc64), ws.wI_rot,
                                  s.lean ? nullptr : ws.wI, ws.Gp64, s.lean ? nullptr : ws.F, s.lean ? ws.fw : nullptr,
                                  ws.priv, c->conv_stream);
  else if (e == cudaSuccess)
    e = mpt::unrotate_tables(s, ws.split_rot, ws.Gc, ws.wI_rot, s.lean ? nullptr : ws.wI, ws.Gp,
                             s.lean ? nullptr : ws.F, s.lean ? ws.fw : nullptr, ws.priv, c->conv_stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->conv_stream);
  if (e != cudaSuccess) st = cuda_fail(c, e, "natural-order tables");
  cudaSetDevice(prev);
  if (st == MPT_OK) c->natural = true;
  return st;
}

// Natural split view: the split table (general path) or the Gc table that the
// conversion wrote it to (blocked path).
const uint32_t* natural_split(const mpt_ctx* c) {
  if (!c->shape.blocked) return c->ws.split;
  return c->shape.wide ? reinterpret_cast<const uint32_t*>(c->ws.Gc64) : c->ws.Gc;
}

}  // namespace

extern "C" {

mpt_status mpt_tables(mpt_ctx* ctx, const int64_t** d_F, const int64_t** d_wI, const uint32_t** d_split) {
  if (!ctx || ctx->tables != MPT_TABLES_INT64) return MPT_ERR_INVALID_ARG;
  if (!ctx->solved) return MPT_ERR_NOT_SOLVED;
  mpt_status st = ensure_natural(ctx);
  if (st != MPT_OK) return st;
  if (d_F) *d_F = ctx->ws.F;
  if (d_wI) *d_wI = ctx->ws.wI;
  if (d_split) *d_split = natural_split(ctx);
  return MPT_OK;
}

mpt_status mpt_tables32(mpt_ctx* ctx, const int32_t** d_F, const uint32_t** d_split) {
  if (!ctx || ctx->tables != MPT_TABLES_LEAN) return MPT_ERR_INVALID_ARG;
  if (!ctx->solved) return MPT_ERR_NOT_SOLVED;
  mpt_status st = ensure_natural(ctx);
  if (st != MPT_OK) return st;
  if (d_F) *d_F = ctx->ws.fw;
  if (d_split) *d_split = natural_split(ctx);
  return MPT_OK;
}

mpt_status mpt_layout_size(const mpt_ctx* ctx, int64_t* total_chunks) {
  if (!ctx || !total_chunks) return MPT_ERR_INVALID_ARG;
  *total_chunks = ctx->shape.slots;
  return MPT_OK;
}

mpt_status mpt_layout(const mpt_ctx* ctx, int64_t* perm_offsets, int64_t* perm_chunks, int32_t* dfs_order) {
  if (!ctx) return MPT_ERR_INVALID_ARG;
  if (!ctx->solved) return MPT_ERR_NOT_SOLVED;
  if (perm_offsets) std::memcpy(perm_offsets, ctx->h_offsets.data(), ctx->h_offsets.size() * 8);
  if (perm_chunks && !ctx->h_chunks.empty()) std::memcpy(perm_chunks, ctx->h_chunks.data(), ctx->h_chunks.size() * 8);
  if (dfs_order) std::memcpy(dfs_order, ctx->h_dfs.data(), ctx->h_dfs.size() * 4);
  return MPT_OK;
}

mpt_status mpt_trie_cost(const int64_t* weights, int64_t n_chunks, int32_t m, const int64_t* perm_offsets,
                         const int64_t* perm_chunks, int64_t* cost) {
  if (!weights || !perm_offsets || !cost || n_chunks < 1 || m < 1) return MPT_ERR_INVALID_ARG;
  if (m > 32) return mpt::trie_cost_lex(weights, n_chunks, m, perm_offsets, perm_chunks, 0, cost);
  if (perm_offsets[0] != 0) return MPT_ERR_INVALID_ARG;
  for (int i = 0; i < m; ++i)
    if (perm_offsets[i + 1] < perm_offsets[i]) return MPT_ERR_INVALID_ARG;
  const int64_t total = perm_offsets[m];
  if (total > 0 && !perm_chunks) return MPT_ERR_INVALID_ARG;
  for (int64_t p = 0; p < total; ++p)
    if (perm_chunks[p] < 0 || perm_chunks[p] >= n_chunks) return MPT_ERR_INVALID_ARG;
  for (int64_t x = 0; x < n_chunks; ++x)
    if (weights[x] <= 0) return MPT_ERR_INVALID_ARG;
  const size_t bw = (size_t)n_chunks * 8, bo = (size_t)(m + 1) * 8, bc = (size_t)(total > 0 ? total : 1) * 8;
  char* d = nullptr;
  if (mpt::device_alloc(reinterpret_cast<void**>(&d), bw + bo + bc + 8) != cudaSuccess) return MPT_ERR_OUT_OF_MEMORY;
  int64_t* dw = reinterpret_cast<int64_t*>(d);
  int64_t* doff = reinterpret_cast<int64_t*>(d + bw);
  int64_t* dch = reinterpret_cast<int64_t*>(d + bw + bo);
  int64_t* dcost = reinterpret_cast<int64_t*>(d + bw + bo + bc);
  mpt_status st = MPT_OK;
  int64_t result = 0;
  if (cudaMemcpy(dw, weights, bw, cudaMemcpyHostToDevice) != cudaSuccess ||
      cudaMemcpy(doff, perm_offsets, bo, cudaMemcpyHostToDevice) != cudaSuccess ||
      (total > 0 && cudaMemcpy(dch, perm_chunks, (size_t)total * 8, cudaMemcpyHostToDevice) != cudaSuccess) ||
      mpt::launch_trie_cost(m, dw, doff, dch, dcost, 0) != cudaSuccess ||
      cudaMemcpy(&result, dcost, 8, cudaMemcpyDeviceToHost) != cudaSuccess) {
    st = MPT_ERR_CUDA;
  }
  cudaFree(d);
  if (st == MPT_OK) *cost = result;
  return st;
}

void mpt_destroy(mpt_ctx* ctx) {
  if (!ctx) return;
  if (ctx->own_ws) cudaFree(ctx->own_ws);
  for (cudaEvent_t e : ctx->events) cudaEventDestroy(e);
  if (ctx->conv_stream) cudaStreamDestroy(ctx->conv_stream);
  delete ctx;
}

}  // extern "C"
