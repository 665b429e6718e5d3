/*
 * CPU oracle for the exact Minimum-Prefix-Trie (MPT) solver.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the independent, slow, plain
 * definition that the CUDA path is checked against.  Only tests/,
 * __graft_entry__.smoke() and bench.py's cpu_baseline leg may load it.  It
 * shares no code, header, table or helper with the CUDA library.
 *
 * What it follows (arxiv 2609.13692, "Prefix Sharing Is a Sorting Problem"):
 *   - Sec. 2: chunks U with weights w(x) >= 1, requests R_1..R_m.  Request i is
 *     bit i of every subset mask.
 *   - Sec. 3 (Thm 1 proof): I(B) is the intersection of R_i over i in B, and
 *     w(I(B)) is the weight of that intersection.
 *   - Sec. 3.1 "Exact algorithm": the savings recurrence
 *       M(B) = w(I(B)) + max over B = B1 (+) B2 of M(B1) + M(B2),
 *     written in cost form F(S) = sum_{i in S} w(R_i) - M(S):
 *       F({i}) = w(R_i),
 *       F(S)   = min over S = A (+) B of F(A) + F(B) - w(I(S)).
 *     OPT_free = F([m]) (Thm 1, eq. 3).
 *
 * Readings where the paper is silent:
 *   - the base case M({i}) = 0, i.e. F({i}) = w(R_i);
 *   - I(empty set) is the set of chunks used by at least one request, so
 *     wI[0] = w(R_1 u ... u R_m); the recurrence never reads it;
 *   - the argmin: every unordered split {A, S\A} is named by the part A that
 *     holds the lowest request index of S; among optimal splits the smallest
 *     such A (as an unsigned integer) is kept.  split[S] = 0 for singletons.
 *
 * Build: gcc -O2 -fopenmp -shared -fPIC oracle.c -o liboracle.so
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ---- intersections (Thm 1 proof: I(B) = intersection of R_i, i in B) ---- */

static int popcount64(uint64_t v) { return __builtin_popcountll(v); }

/* Weight of a chunk bitset over the full universe. */
static int64_t weight_of(const uint64_t* set, int64_t words, int64_t n, const int64_t* w) {
  int64_t total = 0;
  for (int64_t j = 0; j < words; ++j) {
    uint64_t v = set[j];
    while (v) {
      int b = __builtin_ctzll(v);
      int64_t x = j * 64 + b;
      if (x < n) total += w[x];
      v &= v - 1;
    }
  }
  return total;
}

/* w(I(S)) for one subset S, from scratch over the full universe.  For S = 0
 * it returns the weight of the union of all requests (the chunks in play). */
int64_t oracle_wI_one(int32_t m, int64_t n, const int64_t* w, const uint64_t* bits, uint64_t S) {
  int64_t words = (n + 63) / 64;
  uint64_t* acc = (uint64_t*)malloc((size_t)words * sizeof(uint64_t));
  if (!acc) return -1;
  if (S == 0) {
    memset(acc, 0, (size_t)words * sizeof(uint64_t));
    for (int i = 0; i < m; ++i)
      for (int64_t j = 0; j < words; ++j) acc[j] |= bits[(int64_t)i * words + j];
  } else {
    for (int64_t j = 0; j < words; ++j) acc[j] = ~(uint64_t)0;
    for (int i = 0; i < m; ++i) {
      if (!((S >> i) & 1)) continue;
      for (int64_t j = 0; j < words; ++j) acc[j] &= bits[(int64_t)i * words + j];
    }
  }
  int64_t r = weight_of(acc, words, n, w);
  free(acc);
  return r;
}

/* w(I(S)) for every S in [0, 2^m).  The universe is first restricted to the
 * chunks used by some request (no other chunk can lie in an intersection of a
 * non-empty family); then subsets are visited depth-first, each child
 * intersecting its parent's set with one more request. */
typedef struct {
  int m;
  int64_t uw;              /* words of a restricted bitset */
  const uint64_t* req;     /* m rows of uw words: R_i over the used chunks */
  const int64_t* uweight;  /* weight of each used chunk */
  int64_t* wI;
} wi_walk;

static int64_t restricted_weight(const uint64_t* set, int64_t uw, const int64_t* uweight) {
  int64_t total = 0;
  for (int64_t j = 0; j < uw; ++j) {
    uint64_t v = set[j];
    while (v) {
      total += uweight[j * 64 + __builtin_ctzll(v)];
      v &= v - 1;
    }
  }
  return total;
}

static void wi_visit(const wi_walk* c, uint64_t S, int next, const uint64_t* I, uint64_t* stack) {
  /* I is I(S); record it, then extend S by every request index >= next. */
  c->wI[S] = restricted_weight(I, c->uw, c->uweight);
  for (int i = next; i < c->m; ++i) {
    uint64_t* child = stack;
    for (int64_t j = 0; j < c->uw; ++j) child[j] = I[j] & c->req[(int64_t)i * c->uw + j];
    wi_visit(c, S | ((uint64_t)1 << i), i + 1, child, stack + c->uw);
  }
}

int oracle_intersection_weights(int32_t m, int64_t n, const int64_t* w, const uint64_t* bits, int64_t* wI) {
  if (m < 1 || m > 34 || n < 1) return -1;
  int64_t words = (n + 63) / 64;
  /* chunks in play */
  int64_t used = 0;
  for (int64_t x = 0; x < n; ++x) {
    for (int i = 0; i < m; ++i)
      if ((bits[(int64_t)i * words + (x >> 6)] >> (x & 63)) & 1) { ++used; break; }
  }
  int64_t uw = used > 0 ? (used + 63) / 64 : 1;
  uint64_t* req = (uint64_t*)calloc((size_t)(m * uw), sizeof(uint64_t));
  int64_t* uweight = (int64_t*)calloc((size_t)(uw * 64), sizeof(int64_t));
  uint64_t* all = (uint64_t*)calloc((size_t)uw, sizeof(uint64_t));
  uint64_t* stack = (uint64_t*)calloc((size_t)((m + 1) * uw), sizeof(uint64_t));
  if (!req || !uweight || !all || !stack) { free(req); free(uweight); free(all); free(stack); return -2; }
  int64_t u = 0;
  for (int64_t x = 0; x < n; ++x) {
    int in_any = 0;
    for (int i = 0; i < m; ++i) {
      if ((bits[(int64_t)i * words + (x >> 6)] >> (x & 63)) & 1) {
        req[(int64_t)i * uw + (u >> 6)] |= (uint64_t)1 << (u & 63);
        in_any = 1;
      }
    }
    if (in_any) {
      uweight[u] = w[x];
      all[u >> 6] |= (uint64_t)1 << (u & 63);
      ++u;
    }
  }
  wi_walk c = {m, uw, req, uweight, wI};
  wi_visit(&c, 0, 0, all, stack);
  free(req); free(uweight); free(all); free(stack);
  return 0;
}

/* ---- the exact subset recurrence (Sec. 3.1) ---- */

/* Best split of one S (|S| >= 2) from a table F of its proper subsets.
 * A runs over the subsets that hold the lowest request of S, in increasing
 * order, and a later A replaces the incumbent only when strictly cheaper. */
static void best_split(uint64_t S, const int64_t* F, int64_t* best_out, uint64_t* arg_out) {
  uint64_t low = S & (~S + 1);
  uint64_t rest = S ^ low;
  int64_t best = INT64_MAX;
  uint64_t arg = 0;
  uint64_t sub = 0;
  for (;;) {
    if (sub == rest) break; /* A = S is not a split */
    uint64_t A = low | sub;
    int64_t c = F[A] + F[S ^ A];
    if (c < best) { best = c; arg = A; }
    sub = (sub - rest) & rest; /* next larger subset of rest */
  }
  *best_out = best;
  *arg_out = arg;
}

/* Full table: F[S], split[S] for S in [1, 2^m).  F[0] = 0, split[0] = 0.
 * Subsets are finished in order of size, so every F[A], F[S^A] read is final;
 * within one size the subsets are independent and run in parallel. */
int oracle_dp(int32_t m, const int64_t* wI, int64_t* F, uint32_t* split, int32_t nthreads) {
  if (m < 1 || m > 32) return -1;
  uint64_t N = (uint64_t)1 << m;
#ifdef _OPENMP
  if (nthreads > 0) omp_set_num_threads(nthreads);
#else
  (void)nthreads;
#endif
  F[0] = 0;
  split[0] = 0;
  for (int i = 0; i < m; ++i) {
    uint64_t S = (uint64_t)1 << i;
    F[S] = wI[S]; /* F({i}) = w(R_i) */
    split[S] = 0;
  }
  for (int k = 2; k <= m; ++k) {
    int64_t S0;
#pragma omp parallel for schedule(dynamic, 256)
    for (S0 = 1; S0 < (int64_t)N; ++S0) {
      uint64_t S = (uint64_t)S0;
      if (popcount64(S) != k) continue;
      int64_t best;
      uint64_t arg;
      best_split(S, F, &best, &arg);
      F[S] = best - wI[S];
      split[S] = (uint32_t)arg;
    }
  }
  return 0;
}

/* The recurrence's step (Sec. 3.1) at listed subsets only: for each S with
 * |S| >= 2, F(S) and split(S) from the tables F (its proper subsets) and wI,
 * by the same best_split as oracle_dp; subsets with |S| <= 1 get F = wI[S]
 * (0 for S = 0) and split 0.  With the oracle's own tables it reproduces
 * oracle_dp's entries; its use is timing the recurrence on samples of
 * layers too large to finish (each S costs 2^(|S|-1) - 1 splits whatever
 * the table values). */
int oracle_dp_at(int32_t m, const int64_t* wI, const int64_t* F, const uint64_t* subsets, int64_t count,
                 int64_t* F_out, uint32_t* split_out, int32_t nthreads) {
  if (m < 1 || m > 32 || count < 0) return -1;
#ifdef _OPENMP
  if (nthreads > 0) omp_set_num_threads(nthreads);
#else
  (void)nthreads;
#endif
  int64_t t;
#pragma omp parallel for schedule(dynamic, 1)
  for (t = 0; t < count; ++t) {
    uint64_t S = subsets[t];
    if (popcount64(S) <= 1) {
      F_out[t] = (S == 0) ? 0 : wI[S];
      split_out[t] = 0;
      continue;
    }
    int64_t best;
    uint64_t arg;
    best_split(S, F, &best, &arg);
    F_out[t] = best - wI[S];
    split_out[t] = (uint32_t)arg;
  }
  return 0;
}

/* Recompute F(S) and split(S) for a list of subsets from a supplied table
 * (e.g. one produced elsewhere), with w(I(S)) recomputed from scratch.  Used
 * to check sampled entries of tables too large for oracle_dp. */
int oracle_recompute(int32_t m, int64_t n, const int64_t* w, const uint64_t* bits, const int64_t* F_table,
                     const uint64_t* subsets, int64_t count, int64_t* F_out, uint32_t* split_out,
                     int64_t* wI_out, int32_t nthreads) {
#ifdef _OPENMP
  if (nthreads > 0) omp_set_num_threads(nthreads);
#else
  (void)nthreads;
#endif
  int64_t t;
#pragma omp parallel for schedule(dynamic, 1)
  for (t = 0; t < count; ++t) {
    uint64_t S = subsets[t];
    int64_t wi = oracle_wI_one(m, n, w, bits, S);
    wI_out[t] = wi;
    if (popcount64(S) <= 1) {
      F_out[t] = (S == 0) ? 0 : wi;
      split_out[t] = 0;
      continue;
    }
    int64_t best;
    uint64_t arg;
    best_split(S, F_table, &best, &arg);
    F_out[t] = best - wi;
    split_out[t] = (uint32_t)arg;
  }
  return 0;
}

int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
