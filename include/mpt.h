/*
 * mpt.h -- C ABI of the exact Minimum-Prefix-Trie (MPT) solver for GB300 (sm_103a).
 *
 * Problem (arxiv 2609.13692, Sec. 2, eq. 1): a universe of n chunks with
 * positive integer token weights w(x) and m requests R_0..R_{m-1}, each a set
 * of chunks.  Choose, per request, an order of its chunks so that the trie of
 * the resulting strings has the least total weight over its non-root nodes.
 *
 * Method (Thm 1 and Sec. 3.1): the optimum equals a minimum over binary
 * hierarchies on the requests, computed exactly by the subset recurrence
 *     F({i}) = w(R_i),
 *     F(S)   = min over S = A (+) B of F(A) + F(B) - w(I(S)),
 * where I(S) is the intersection of R_i over i in S.  OPT = F({0..m-1}).
 * All work runs in CUDA kernels on the caller's stream; the host only
 * validates arguments and orders launches.
 *
 * Conventions shared by every call:
 *   - Request i is bit i of every subset mask (request 0 = least significant).
 *   - Request bitsets: uint64 row-major [m][ceil(n/64)]; bit (x % 64) of word
 *     (x / 64) in row i is set iff chunk x is in R_i.
 *   - Chunk ids in every output are the caller's ids 0..n-1.
 *   - Among optimal splits of S, the reported one is named by its part A that
 *     holds the lowest request of S, and the smallest such A (as an unsigned
 *     integer) is chosen; split[S] = A, 0 for singletons and for S = 0.
 *   - Every call returns a status; on failure no output is written.
 *   - A context is not thread-safe; distinct contexts are independent.
 *   - Limits: 1 <= m <= 32, 1 <= n <= 2^31 - 1, every w(x) >= 1, and
 *     sum_i w(R_i) < 2^62 (MPT_ERR_OVERFLOW otherwise).
 */
#ifndef MPT_H
#define MPT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum mpt_status {
  MPT_OK = 0,
  MPT_ERR_INVALID_ARG = 1,         /* null pointer, m < 1, n < 1, w(x) <= 0, a bit set at x >= n */
  MPT_ERR_TOO_LARGE = 2,           /* beyond a documented limit (m > 32 for mpt_create) */
  MPT_ERR_OVERFLOW = 3,            /* sum_i w(R_i) >= 2^62 */
  MPT_ERR_OUT_OF_MEMORY = 4,       /* host or device allocation failed */
  MPT_ERR_WORKSPACE_TOO_SMALL = 5, /* caller workspace below mpt_workspace_bytes() */
  MPT_ERR_CUDA = 6,                /* a CUDA call failed; mpt_last_error() has its text */
  MPT_ERR_NOT_SOLVED = 7,          /* results asked for before a successful mpt_solve */
  MPT_ERR_TIMEOUT = 8,             /* a bounded wait on a shared-memory barrier inside a kernel gave up */
  MPT_ERR_INTERNAL = 9             /* a device-side consistency check failed */
} mpt_status;

typedef struct mpt_ctx mpt_ctx;

/* DP kernels mpt_solve may use.  Their limits are on the shared weight
 * W = sum_i w(R_i) - sum_i pi_i - m u, where pi_i is the weight of the
 * chunks that request i alone needs and u (m >= 2) that of the chunks every
 * request needs.  Such a chunk is one cluster in every hierarchy (t_x(H) = 1
 * in Thm 1): it adds w(x) to F(S) for every non-empty S holding its
 * requests, whatever the splits.  The tiled kernels therefore run the
 * recurrence on F(S) - sum_{i in S} pi_i - u and add it back in every output.
 * AUTO picks BLOCKED whenever W < 2^(32 - b), b = min(m, 12) tile bits
 * (2^20 from m = 12 on; its 32-bit packed keys are then exact), else WIDE
 * while W < 2^51 (64-bit packed keys), else GENERAL.  All of them return the
 * same tables, OPT and layout. */
typedef enum mpt_dp_mode {
  MPT_DP_AUTO = 0,
  MPT_DP_BLOCKED = 1, /* shared-memory tiled min-plus; needs W < 2^(32 - min(m, 12)) */
  MPT_DP_GENERAL = 2, /* one subset per thread or warp, int64 gathers from HBM/L2 */
  MPT_DP_WIDE = 3     /* the tiled min-plus with 64-bit keys; needs W < 2^51 */
} mpt_dp_mode;

/* Create a context for one instance (Sec. 2).
 *   weights:  host int64[n_chunks], w(x) >= 1 for every x.
 *   req_bits: host uint64[m][ceil(n_chunks/64)], as above; no bit at x >= n.
 * Both arrays are validated and copied; the caller keeps ownership.
 * Errors: INVALID_ARG, TOO_LARGE, OVERFLOW, OUT_OF_MEMORY.  *out is written
 * only on success.  No CUDA call is made. */
mpt_status mpt_create(const int64_t* weights, int64_t n_chunks, const uint64_t* req_bits, int32_t m,
                      mpt_ctx** out);

/* Bytes of device workspace mpt_solve needs for this context: the input
 * copies, the intersection-weight table wI int64[2^m], F int64[2^m],
 * split uint32[2^m], the blocked DP's working tables and the layout buffers. */
mpt_status mpt_workspace_bytes(const mpt_ctx* ctx, size_t* bytes);

/* Choose the DP kernels (default MPT_DP_AUTO).  BLOCKED is refused with
 * OVERFLOW when the shared weight W (above) is >= 2^(32 - min(m, 12)), WIDE
 * when W >= 2^51. */
mpt_status mpt_set_dp_mode(mpt_ctx* ctx, int32_t mode);

/* Solve exactly (Sec. 3.1): scatter chunk weights by request set, superset
 * sums for w(I(S)) of every S, the popcount-layered min-plus recurrence with
 * its argmin table, then the hierarchy walk for the layout (Thm 1 proof).
 *   d_workspace: device memory of at least mpt_workspace_bytes(), 256-byte
 *     aligned, owned by the caller.  Nothing else may write it while this
 *     context uses it: the instance copied into it by one solve is reused
 *     (not copied again) by the next solve of the same context with the same
 *     workspace.  NULL makes the library allocate (and keep) its own.
 *   stream: a cudaStream_t (NULL = the legacy default stream).  Every copy
 *     and kernel is enqueued on it; the call synchronises it before return.
 *   opt_cost: host int64, receives OPT = F({0..m-1}).
 * Errors: INVALID_ARG, WORKSPACE_TOO_SMALL, OUT_OF_MEMORY, CUDA, INTERNAL. */
mpt_status mpt_solve(mpt_ctx* ctx, void* d_workspace, size_t workspace_bytes, void* stream, int64_t* opt_cost);

/* Staged solve: the same computation as mpt_solve in resumable pieces, for
 * long solves (m = 31..32 runs for tens of seconds) that must yield the GPU,
 * report progress or survive a restart.  The recurrence runs in steps that
 * each depend only on earlier ones (Sec. 3.1 layers: one step per tile layer
 * |T| = 0 .. m - b of the blocked kernels, or the singletons and one step per
 * subset size of the general kernels); mpt_solve_steps gives their number.
 *   mpt_solve_begin:  input copies, K1, K2 and step 0;
 *   mpt_solve_layers: the next `count` steps (fewer at the end); *next_step
 *                     (may be NULL) receives the index of the next step;
 *   mpt_solve_end:    after the last step: the layout walk and OPT, as
 *                     mpt_solve (then mpt_tables / mpt_layout apply).
 * Every call enqueues its work on `stream` and returns (mpt_solve_end
 * synchronises it).  Between calls the workspace holds the whole state: once
 * the stream is idle, a copy of its mpt_workspace_bytes() bytes is a
 * checkpoint.  To resume, copy it back into a workspace (any 256-byte-aligned
 * device buffer of that size) and call mpt_solve_resume with the step the
 * checkpoint had reached, on a context created from the same instance with
 * the same DP mode and table layout.  All three step calls must name the same workspace
 * (NULL: the context's own, for begin, layers and end only).
 * Errors: INVALID_ARG (wrong workspace, step out of range), NOT_SOLVED (no
 * staged solve begun, or steps left before mpt_solve_end), and those of
 * mpt_solve. */
mpt_status mpt_solve_steps(const mpt_ctx* ctx, int32_t* steps);
mpt_status mpt_solve_begin(mpt_ctx* ctx, void* d_workspace, size_t workspace_bytes, void* stream);
mpt_status mpt_solve_layers(mpt_ctx* ctx, void* d_workspace, size_t workspace_bytes, void* stream, int32_t count,
                            int32_t* next_step);
mpt_status mpt_solve_end(mpt_ctx* ctx, void* d_workspace, size_t workspace_bytes, void* stream, int64_t* opt_cost);
mpt_status mpt_solve_resume(mpt_ctx* ctx, void* d_workspace, size_t workspace_bytes, int32_t next_step);

/* Device views (length 2^m, indexed by subset mask S) of the last solve:
 *   F[S]     = the recurrence value (F[0] = 0),
 *   wI[S]    = w(I(S)); wI[0] = weight of the union of all requests,
 *   split[S] = the reported optimal split (see conventions).
 * The pointers live in the workspace and stay valid until the next solve or
 * mpt_destroy.  Any argument may be NULL.  The blocked recurrence keeps its
 * tables in a tile-major (rotated) order; the first call after such a solve
 * writes the natural-order views inside the workspace (a transpose of about
 * 36 bytes per subset, ~1.5 ms at m = 28) on a stream of the context, on the
 * device of the solve, and waits for it; later calls only return the
 * pointers.  Errors: INVALID_ARG (also when the context uses
 * MPT_TABLES_LEAN: see mpt_tables32), NOT_SOLVED, CUDA. */
mpt_status mpt_tables(mpt_ctx* ctx, const int64_t** d_F, const int64_t** d_wI, const uint32_t** d_split);

/* Table layout of the solve (Sec. 3.1 tables; N3 "leaner" form).
 *   MPT_TABLES_INT64 (default): w(I(S)) and F(S) in separate int64[2^m]
 *     tables (mpt_tables);
 *   MPT_TABLES_LEAN: one int32[2^m] table that holds w(I(S)) after K2 and
 *     F(S) afterwards (general path: each entry is overwritten in place by
 *     the thread that finishes it; blocked path: F is written over it when
 *     mpt_tables32 asks for the natural views), read with mpt_tables32;
 *     w(I(S)) is then no longer available.  Allowed when sum_i w(R_i) < 2^31
 *     (MPT_ERR_OVERFLOW otherwise), which bounds every w(I(S)) and F(S).
 *     The blocked path's workspace falls from 28 to 16 bytes per subset
 *     (m = 32: 64 GiB instead of 112 GiB).
 * Changing the layout discards the last solve.  Errors: INVALID_ARG, OVERFLOW. */
#define MPT_TABLES_INT64 0
#define MPT_TABLES_LEAN 1
mpt_status mpt_set_tables(mpt_ctx* ctx, int32_t kind);

/* Device views of the lean tables of the last solve: F int32[2^m] and split
 * uint32[2^m] (as in mpt_tables, including the conversion on the first call).
 * Errors: INVALID_ARG (not lean), NOT_SOLVED, CUDA. */
mpt_status mpt_tables32(mpt_ctx* ctx, const int32_t** d_F, const uint32_t** d_split);

/* Number of entries mpt_layout writes to perm_chunks: sum_i |R_i|. */
mpt_status mpt_layout_size(const mpt_ctx* ctx, int64_t* total_chunks);

/* Layout of the last solve (constructive direction of Thm 1): at hierarchy
 * node B (root = all requests, children split[B] then B \ split[B]) the chunks
 * of I(B) \ I(parent(B)) are emitted in increasing chunk id; request i's
 * permutation is the concatenation along its root-to-leaf path.
 *   perm_offsets: host int64[m+1]; request i is perm_chunks[off[i] .. off[i+1]).
 *   perm_chunks:  host int64[mpt_layout_size()].
 *   dfs_order:    host int32[m], the leaves from left to right -- the serving
 *                 order of Thm 7 (Sec. 8).
 * Any output may be NULL.  Errors: INVALID_ARG, NOT_SOLVED. */
mpt_status mpt_layout(const mpt_ctx* ctx, int64_t* perm_offsets, int64_t* perm_chunks, int32_t* dfs_order);

/* Trie cost of a layout (Sec. 2, eq. 1): the total weight of the non-root
 * nodes of the trie of the m strings, computed on the GPU.  All pointers are
 * host memory; perm_offsets has m+1 entries, perm_chunks perm_offsets[m]
 * entries with ids in [0, n_chunks).  Up to 32 strings one block compares
 * every pair; beyond that the strings are sorted lexicographically and each
 * adds the weight of its suffix after the common prefix with its predecessor.
 * Limits: m <= 2^22 strings, perm_offsets[m] <= 2^27, each string <= 4096
 * chunks (MPT_ERR_TOO_LARGE).  The call allocates and frees a device buffer
 * and synchronises the legacy default stream.
 * Errors: INVALID_ARG, TOO_LARGE, OUT_OF_MEMORY, CUDA. */
mpt_status mpt_trie_cost(const int64_t* weights, int64_t n_chunks, int32_t m, const int64_t* perm_offsets,
                         const int64_t* perm_chunks, int64_t* cost);

/* Per-stage device timings of the last solve, taken with CUDA events on the
 * solve's stream when profiling is on (mpt_set_profiling). */
typedef struct mpt_profile {
  double ms_h2d;        /* input copies */
  double ms_scatter;    /* N_x and g(T) scatter */
  double ms_zeta;       /* superset sums -> wI */
  double ms_dp_pairs;   /* blocked DP: all launches of the pair kernel */
  double ms_dp_tiles;   /* blocked DP: all launches of the in-tile kernel */
  double ms_dp_general; /* general DP: all launches */
  double ms_walk;       /* hierarchy walk -> layout */
  double ms_d2h;        /* result copies */
  double splits_pairs;  /* splits evaluated by the pair kernel */
  double splits_total;  /* (3^m + 1)/2 - 2^m */
  int64_t launches_pairs;
  int64_t launches_total; /* kernels launched by the last solve (memsets excluded) */
  int32_t dp_mode;        /* MPT_DP_BLOCKED, MPT_DP_WIDE or MPT_DP_GENERAL as used */
  int32_t tile_bits;      /* request bits per shared-memory tile (blocked mode) */
} mpt_profile;

mpt_status mpt_set_profiling(mpt_ctx* ctx, int32_t on);
mpt_status mpt_get_profile(const mpt_ctx* ctx, mpt_profile* out);

/* ---------------------------------------------------------------------------
 * Batched exact solves of many small instances (the paper's own use of the
 * recurrence: synthetic groups of 10-15 requests, Sec. 6.2, and real request
 * groups of at most 13, Sec. 7); instances of up to 16 requests.
 * Every instance shares one chunk universe and weight array; instance b owns
 * requests inst_requests[b] .. inst_requests[b+1]-1, request r the chunk ids
 * chunk_ids[req_offsets[r] .. req_offsets[r+1]).  One CUDA block solves one
 * instance with all of its tables in shared memory; results follow the same
 * conventions as mpt_solve / mpt_layout for each instance on its own (request
 * bit i = the instance's i-th request).
 * ------------------------------------------------------------------------- */
typedef struct mpt_batch mpt_batch;

/* Validate and copy a batch (host arrays; caller keeps ownership).
 *   weights: int64[n_chunks] (>= 1); inst_requests: int64[batch+1], starting at
 *   0; req_offsets: int64[inst_requests[batch]+1], starting at 0;
 *   chunk_ids: int64[req_offsets[last]] in [0, n_chunks), no repeat inside a
 *   request.
 * Limits per instance: 1 <= m <= 16 and at most 2048 chunk occurrences
 * (1024 at m = 15 unless the keys pack, see below; at m = 16 the keys must
 * pack: shared weight below 2^16; MPT_ERR_TOO_LARGE beyond); sum_i w(R_i) < 2^62 and a shared weight
 * (sum_i w(R_i) less the chunks that one request alone or all m >= 2
 * requests hold, see MPT_DP_AUTO) below 2^31 (MPT_ERR_OVERFLOW).
 * Errors: INVALID_ARG, TOO_LARGE, OVERFLOW, OUT_OF_MEMORY.  No CUDA call. */
mpt_status mpt_batch_create(const int64_t* weights, int64_t n_chunks, int32_t batch, const int64_t* inst_requests,
                            const int64_t* req_offsets, const int64_t* chunk_ids, mpt_batch** out);

/* Device workspace bytes of mpt_batch_solve: input copies, per-instance
 * F int64 / split uint32 tables (sum over instances of 2^m entries), OPT,
 * permutations and DFS orders. */
mpt_status mpt_batch_workspace_bytes(const mpt_batch* b, size_t* bytes);

/* Solve every instance (Sec. 3.1 recurrence and Thm 1 layout per instance).
 * d_workspace as in mpt_solve (NULL: the library allocates and keeps one).
 * Uploads and downloads run on `stream`; the per-size grids run on four
 * side streams of the batch object (created on the first solve, on the
 * device current then, and released by mpt_batch_destroy), forked from
 * `stream` after the uploads and joined back to it before the downloads;
 * `stream` is synchronised before return, so no work of the call outlives
 * it.  If the side streams cannot be created the grids run on `stream`.
 * Errors: INVALID_ARG, WORKSPACE_TOO_SMALL, OUT_OF_MEMORY, CUDA, INTERNAL. */
mpt_status mpt_batch_solve(mpt_batch* b, void* d_workspace, size_t workspace_bytes, void* stream);

/* Results of the last solve, host outputs (any may be NULL):
 *   opt: int64[batch];
 *   perm_chunks: int64[req_offsets[last]], each request's chunks in layout
 *     order, in the request's own slot range of the input CSR;
 *   dfs_order: int32[inst_requests[batch]], per instance the local request
 *     indices (0..m-1) from left to right (Thm 7 serving order).
 * Errors: INVALID_ARG, NOT_SOLVED. */
mpt_status mpt_batch_results(const mpt_batch* b, int64_t* opt, int64_t* perm_chunks, int32_t* dfs_order);

/* Device tables of the last solve: instance b's F and split (indexed by its
 * local subset masks) start at table_offsets[b] (host int64[batch+1]).
 * Valid until the next solve or destroy.  Errors: INVALID_ARG, NOT_SOLVED. */
mpt_status mpt_batch_tables(const mpt_batch* b, const int64_t** d_F, const uint32_t** d_split,
                            int64_t* table_offsets);

/* Releases the batch, its library-owned workspace and its side streams.  A
 * batch object, like a context, is not thread-safe; distinct batches are
 * independent. */
void mpt_batch_destroy(mpt_batch* b);

/* Agglomerative common-intersection hierarchy (Sec. 6.2; H_g of Thm 6) and
 * the spanning-tree lower bound (Sec. 6.3), for request counts far beyond the
 * exact recurrence.  Every request starts as a cluster with signature R_i;
 * the two active clusters with the heaviest common signature merge, the
 * merged signature being that intersection.  A cluster lives in the slot of
 * its smallest request; ties go to the smallest slot pair (a, b), a < b, and
 * the merged cluster keeps slot a.  The layout walks the hierarchy top-down
 * as in the Thm 1 proof (children of a merge: slot a's subtree first).
 *   weights: host int64[n_chunks] (>= 1); req_offsets: host int64[m+1] from 0;
 *   chunk_ids: host int64[req_offsets[m]], at most 128 per request, no repeat
 *   inside a request, each request's weight < 2^32.  1 <= m <= 16384.
 *   stream: a cudaStream_t (NULL = legacy default), synchronised before return.
 * Outputs (host, any may be NULL): cost = sum_i w(R_i) - savings (the
 * hierarchy's Thm 1 cost; the trie of the layout costs at most this),
 * savings = sum of merge values, lower_bound = sum_i w(R_i) - max spanning
 * tree of w(R_i cap R_j), merges int32[2(m-1)] (slot pairs a, b in merge
 * order), merge_values int64[m-1], perm_chunks int64[req_offsets[m]] (each
 * request's chunks in layout order, in its own CSR range), dfs_order int32[m].
 * Device memory (m^2 * 4 bytes for the pair weights, plus small buffers) is
 * allocated and freed by the call.
 * Errors: INVALID_ARG, TOO_LARGE, OVERFLOW, OUT_OF_MEMORY, CUDA. */
mpt_status mpt_greedy(const int64_t* weights, int64_t n_chunks, int32_t m, const int64_t* req_offsets,
                      const int64_t* chunk_ids, void* stream, int64_t* cost, int64_t* savings,
                      int64_t* lower_bound, int32_t* merges, int64_t* merge_values, int64_t* perm_chunks,
                      int32_t* dfs_order);

/* ---------------------------------------------------------------------------
 * Serving order and finite cache (Sec. 8, Thm 7)
 *
 * Strings are laid-out requests, given as a host CSR: string i is
 * seq_chunks[seq_offsets[i] .. seq_offsets[i+1]) (chunk ids in [0, n_chunks);
 * seq_offsets[0] = 0).  Limits: 1 <= m <= 2^22 strings, seq_offsets[m] <=
 * 2^27 chunk occurrences, each string <= 4096 chunks (MPT_ERR_TOO_LARGE).
 * Each call allocates and frees its device buffers, runs on `stream` (a
 * cudaStream_t, NULL = legacy default) and synchronises it before returning.
 * ------------------------------------------------------------------------- */

/* Thm 7's serving order: the strings sorted lexicographically (a string
 * before its extensions; identical strings by increasing index), which is the
 * DFS order of their trie.  With 0 < window < m, the stream `arrival` (a
 * permutation of 0..m-1, NULL = 0, 1, .., m-1) is cut into consecutive
 * windows of `window` arrivals and each window is sorted on its own -- the
 * bounded reorder window of Sec. 8.1; window = 0 or >= m sorts everything.
 *   order: host int32[m], the request served at each position.
 * Errors: INVALID_ARG, TOO_LARGE, OUT_OF_MEMORY, CUDA. */
mpt_status mpt_serve_order(int64_t n_chunks, int32_t m, const int64_t* seq_offsets, const int64_t* seq_chunks,
                           const int32_t* arrival, int32_t window, void* stream, int32_t* order);

/* Prefill cost under a finite radix (prefix) cache, for several capacities at
 * once (Sec. 8).  Requests are served in `order` (host int32[m], a
 * permutation; NULL = 0, 1, .., m-1).  The cache holds trie nodes (one chunk
 * each, weight w(chunk)); a cached node implies its ancestors are cached.
 * Serving a request computes, and pays for, every chunk of its string past
 * the longest cached prefix, then inserts them; when the cached weight exceeds
 * the capacity, least recently used leaves that are not on the current
 * request's path are evicted (a request touches every node of its path), and
 * chunks that still find no room are computed without being cached.
 *   weights: host int64[n_chunks] (>= 1); capacities: host int64[n_caps]
 *   (>= 0, n_caps <= 1024);
 *   costs: host int64[n_caps], the total prefill weight at each capacity;
 *   unbounded: host int64[1] (may be NULL), the cost with no eviction = the
 *   trie weight of eq. (1).
 * Thm 7: in the order of mpt_serve_order, any capacity >= max_i w(string i)
 * pays exactly `unbounded`.  Errors: INVALID_ARG, TOO_LARGE, OVERFLOW (total
 * string weight >= 2^62), OUT_OF_MEMORY, CUDA, INTERNAL. */
mpt_status mpt_cache_costs(const int64_t* weights, int64_t n_chunks, int32_t m, const int64_t* seq_offsets,
                           const int64_t* seq_chunks, const int32_t* order, const int64_t* capacities,
                           int32_t n_caps, void* stream, int64_t* costs, int64_t* unbounded);

/* Quality-preserving variant of the layout (Sec. 7.1): each request's t most
 * relevant passages are pinned at the end of its prompt, in relevance order
 * (rank 1 first), and only the rest is laid out: by the exact recurrence
 * (method MPT_PIN_EXACT, m <= 32) or by the agglomerative hierarchy
 * (MPT_PIN_GREEDY, the limits of mpt_greedy) on the reduced request sets.
 *   ranked_offsets / ranked_chunks: host CSR, request i's passages in
 *   relevance order (most relevant first), no repeats inside a request;
 *   t >= 0 (a request with at most t passages is pinned whole);
 *   perm_chunks: host int64[ranked_offsets[m]] (may be NULL), each request's
 *   laid-out string in its own CSR range;
 *   serve_order: host int32[m] (may be NULL), Thm 7's order of those strings;
 *   cost: host int64[1] (may be NULL), their trie weight (eq. 1).
 * Errors: those of mpt_create / mpt_solve or mpt_greedy, plus INVALID_ARG and
 * TOO_LARGE. */
#define MPT_PIN_EXACT 0
#define MPT_PIN_GREEDY 1
mpt_status mpt_layout_pinned(const int64_t* weights, int64_t n_chunks, int32_t m, const int64_t* ranked_offsets,
                             const int64_t* ranked_chunks, int32_t t, int32_t method, void* stream,
                             int64_t* perm_chunks, int32_t* serve_order, int64_t* cost);

/* Exact solve that allocates nothing, for callers that cannot allocate device
 * memory: code running in a serving process whose device memory is reserved
 * up front by its own pool allocator, or code that must not call cudaMalloc /
 * cudaFree because those calls synchronise the device and stall the work
 * already running on it.  The paper has no counterpart; it is a deployment
 * variant of mpt_solve that returns the tables and OPT but no layout.
 *   d_weights:  device int64[n_chunks];  d_req_bits: device uint64[m][ceil(n/64)]
 *   d_F, d_wI:  device int64[2^m];       d_split:    device uint32[2^m]
 *   d_opt:      device int64[1]          (all caller-owned; same meaning as
 *               mpt_tables and mpt_solve's OPT)
 *   stream:     a cudaStream_t (NULL = the legacy default stream).
 * Limits: m <= 20 and sum_i |R_i| <= 65536 (MPT_ERR_TOO_LARGE beyond),
 * w(x) >= 1 and no bit at x >= n (MPT_ERR_INVALID_ARG), sum_i w(R_i) < 2^62
 * (MPT_ERR_OVERFLOW).  The scratch -- the blocked recurrence's working tables
 * and per-layer minima -- is one file-scope device array of 10.7 MiB that
 * every GPU loading this library holds until the process exits.  The first
 * call on a device looks up that array's device address (and the device's
 * SM count) and keeps it for the life of the process, so make it before any
 * stream capture, and do not reset the device (cudaDeviceReset) while the
 * library is loaded.  Every call synchronises `stream` once, to read the
 * input check, then enqueues the solve and returns: the outputs are ready
 * when the stream reaches that point.  The device-side consistency flags
 * that mpt_solve reports as MPT_ERR_INTERNAL are not read back by this call.
 * Every call shares the one array and finds the previous call's contents in
 * it; calls whose work overlaps on the GPU (other streams, other host
 * threads) race and must be serialised. */
mpt_status mpt_solve_noalloc(const int64_t* d_weights, int64_t n_chunks, const uint64_t* d_req_bits, int32_t m,
                             int64_t* d_F, int64_t* d_wI, uint32_t* d_split, int64_t* d_opt, void* stream);

/* Measurement helper, not part of the method: the useful bandwidth of
 * uniformly random, independent 8-byte loads from a table of 2^log2_entries
 * int64 entries -- the access pattern of the Sec. 3.1 recurrence without
 * blocking (two table reads per split).  About `loads` loads (indices from a
 * counter-based hash) are timed with CUDA events on `stream` after one
 * warm-up pass; the table is allocated, filled and freed by the call on the
 * current device.  gbps: 8 bytes per load / elapsed seconds / 1e9.
 * 10 <= log2_entries <= 32.  Errors: INVALID_ARG, OUT_OF_MEMORY, CUDA. */
mpt_status mpt_gather_bandwidth(int32_t log2_entries, int64_t loads, void* stream, double* gbps);

/* Measurement helper, not part of the method: the measured peak rate of the
 * one instruction the blocked Sec. 3.1 recurrence issues per split -- a
 * 32-bit add fused with an unsigned min, acc = min(acc, x + y), on the
 * integer ALU pipe -- with every SM busy (16 warps each, 32 independent
 * minima per thread, no memory traffic in the loop).  About `ops` add-mins
 * are timed with CUDA events on `stream` after a short warm-up launch.
 * ops_per_s: add-mins per second at whatever SM clock the GPU ran (the
 * caller samples it); the nominal figure is SMs x 64 lanes x clock.
 * 1 <= ops < ~2^28 x SMs x 2^19.  Errors: INVALID_ARG, OUT_OF_MEMORY (an
 * 8-byte sink), CUDA. */
mpt_status mpt_alu_addmin_peak(int64_t ops, void* stream, double* ops_per_s);

/* How this copy of the library was built, as bits in *flags: bit 0 set
 * means the bounds-checked variant (compiled with MPT_BOUNDS), whose kernels
 * test table indices, window offsets and split entries, skip any access that
 * fails and report MPT_ERR_INTERNAL from mpt_solve -- a stand-in for a
 * device memory checker, slower than the default build.  Not part of the
 * method.  Errors: INVALID_ARG (flags NULL). */
mpt_status mpt_build_info(int32_t* flags);

/* Free the context and any workspace the library allocated.  NULL is a no-op. */
void mpt_destroy(mpt_ctx* ctx);

/* Static text for a status code. */
const char* mpt_status_string(mpt_status status);

/* Text of the last CUDA or internal error seen by this context ("" if none). */
const char* mpt_last_error(const mpt_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* MPT_H */
