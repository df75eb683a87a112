/*
 * wl.h -- seeded synthetic workload generator for the prefix-cache-aware router.
 *
 * This module is the one input source shared by the CPU oracle and the CUDA path.  It produces token
 * sequences (the contents of each peer's radix tree), request batches, peer loads and ordered
 * INSERT/DELETE deltas.  It contains no radix-tree or routing arithmetic: it only draws random numbers
 * and keeps, per tree, the list of sequence identities that are currently stored.
 *
 * Workload model (stand-in for the few-shot-prompt workloads of the paper's Section 4: topic prompts that
 * share a long few-shot prefix, with a skewed topic popularity):
 *   - n_prefix shared prefixes, lengths uniform [pre_lo, pre_hi], tokens uniform [0, vocab).
 *   - each prefix is assigned to each tree independently with probability assign_prob.
 *   - a tree sequence = one of the tree's assigned prefixes, chosen with Zipf(zipf_s) weights renormalised
 *     over the assigned set (rank = prefix index), followed by a random suffix of length [suf_lo, suf_hi].
 *   - a request = a prefix chosen Zipf(zipf_s) over all prefixes followed by a random suffix of length
 *     [req_suf_lo, req_suf_hi]; with probability fresh_frac the prefix is a fresh random one instead.
 *     With diverge=1 (long-context case) a shared request is prefix[:d] + one token != prefix[d] + a
 *     random tail, d uniform in [0, len-1].
 *   - load[p] uniform [0, load_hi].
 *
 * Sequences are handed out in "segmented" form: a sequence is the concatenation of one or more
 * (offset, length) runs in a token pool.  The pool of every tree/delta fill starts with the shared
 * prefix table (wl_prefix_pool), followed by the suffix tokens of that fill.
 *
 * PRNG: SplitMix64 (to seed) and xoshiro256** (Blackman & Vigna, 2018); bounded integers by Lemire's
 * multiply-shift method (2019); Zipf by inverse CDF over a cumulative table.  Every random quantity is
 * derived from a stream keyed by (seed, tag, i, j), so fills are independent of call order and threads.
 */
#ifndef P2P_WORKLOAD_WL_H
#define P2P_WORKLOAD_WL_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct wl_params {
  int32_t P;              /* number of trees (peers) */
  int32_t vocab;          /* tokens are uniform in [0, vocab) */
  int64_t n_seq;          /* sequences inserted into each tree */
  int32_t n_prefix;       /* shared prefixes */
  int32_t pre_lo, pre_hi; /* prefix length range, inclusive */
  int32_t suf_lo, suf_hi; /* tree-sequence suffix length range, inclusive */
  double zipf_s;          /* Zipf exponent of prefix popularity */
  double assign_prob;     /* probability that a prefix is cached in a given tree */
  int64_t B;              /* requests per batch */
  double fresh_frac;      /* share of requests with a fresh (uncached) random prefix */
  int32_t req_suf_lo, req_suf_hi; /* request suffix / tail length range */
  int32_t diverge;        /* 1: shared requests diverge at a uniform random depth inside the prefix */
  int32_t load_hi;        /* load uniform in [0, load_hi] */
  int32_t alpha;          /* load weight in the route score */
  double stale_del_frac;  /* trees p >= 1: share of stored sequences dropped from the replica */
  double stale_ins_frac;  /* trees p >= 1: extra sequences (share of n_seq) only in the replica */
  double delta_frac;      /* per-batch delta: ceil(delta_frac * live) DELETEs and as many INSERTs */
} wl_params;

typedef struct wl_gen wl_gen;

/* Fills the preset for workload id 0..4; returns 0, or -1 for an unknown id. */
int wl_preset(int32_t cfg_id, wl_params* out);
/* Default seed of workload id c: 0x9E3779B97F4A7C15 xor c. */
uint64_t wl_default_seed(int32_t cfg_id);

/* Creates a generator (prefix table, assignments, per-tree sequence lists; for stale replicas also the
 * replica lists and the delta that turns the exact tree into the replica).  NULL on bad parameters. */
wl_gen* wl_create(const wl_params* prm, uint64_t seed);
void wl_free(wl_gen* g);
void wl_get_params(const wl_gen* g, wl_params* out);

/* The shared prefix table: n_prefix runs; wl_prefix_pool copies all prefix tokens (n_pool_tokens) and the
 * start offset / length of every prefix.  Every pool filled below starts with this table. */
int64_t wl_prefix_pool_size(const wl_gen* g);
void wl_prefix_pool(const wl_gen* g, int32_t* pool, int64_t* pre_off, int32_t* pre_len);

/* Tree contents.  which = 0: the tree's current sequence list (the replica); which = 1: the exact tree
 * (differs from 0 only for stale replicas, before any delta).  size: number of sequences, segments and
 * suffix tokens.  fill: seg_begin[n+1], seg_off[n_segs], seg_len[n_segs] and the suffix tokens, which are
 * written at suffix_out and referenced at pool offset suffix_base (normally wl_prefix_pool_size). */
int wl_tree_size(const wl_gen* g, int32_t p, int32_t which, int64_t* n_seq, int64_t* n_segs, int64_t* n_suffix_tokens);
int wl_tree_fill(const wl_gen* g, int32_t p, int32_t which, int64_t* seg_begin, int64_t* seg_off,
                 int32_t* seg_len, int32_t* suffix_out, int64_t suffix_base);

/* Requests [b0, b1) as a plain CSR: total token count, then tokens and offsets[b1-b0+1] (offsets[0]=0).
 * Threads split the range; results do not depend on n_threads. */
int64_t wl_requests_size(const wl_gen* g, int64_t b0, int64_t b1, int32_t n_threads);
int wl_requests_fill(const wl_gen* g, int64_t b0, int64_t b1, int32_t* tokens, int64_t* offsets, int32_t n_threads);

/* load[P] for batch `step` (the same for every step unless vary_per_step). */
int wl_load_fill(const wl_gen* g, int64_t step, int32_t vary_per_step, int32_t* load);

/* Deltas.  wl_delta_make draws, for every tree p in [p0, p1), ceil(del_frac * live) DELETEs of distinct
 * stored sequences and ceil(ins_frac * live) INSERTs of new sequences (randomly interleaved), updates the
 * tree's sequence list, and keeps the ops as the tree's pending delta.  Seeded by (seed, step, p).
 * Op codes: 0 = INSERT, 1 = DELETE.  wl_delta_size / wl_delta_fill hand out the pending deltas of trees
 * [p0, p1) concatenated, with peer_begin[p1-p0+1] marking each tree's op range.  For stale replicas the
 * pending delta after wl_create is the exact-tree -> replica delta. */
int wl_delta_make(wl_gen* g, int32_t p0, int32_t p1, int64_t step, double del_frac, double ins_frac, int32_t n_threads);
int wl_delta_size(const wl_gen* g, int32_t p0, int32_t p1, int64_t* n_ops, int64_t* n_segs, int64_t* n_suffix_tokens);
int wl_delta_fill(const wl_gen* g, int32_t p0, int32_t p1, int32_t* op, int64_t* seg_begin, int64_t* seg_off,
                  int32_t* seg_len, int32_t* suffix_out, int64_t suffix_base, int64_t* peer_begin, int32_t n_threads);

/* Raw PRNG access, for tests of the published generators. */
uint64_t wl_splitmix64(uint64_t* state);
void wl_xoshiro_seed(uint64_t seed, uint64_t s[4]);
uint64_t wl_xoshiro_next(uint64_t s[4]);
uint64_t wl_bounded(uint64_t s[4], uint64_t range);
/* Zipf draw over n ranks with exponent s from a 53-bit uniform u in [0,1): smallest k with cdf(k) > u. */
int32_t wl_zipf_index(int32_t n, double s, double u);

#ifdef __cplusplus
}
#endif
#endif
