/*
 * p2p_router.h -- C ABI of the GB300 batched routing engine for decentralized, prefix-cache-aware routing
 * ("Towards Distributed Inference of LLMs on a P2P Network").
 *
 * A router holds P radix trees in GPU memory: by convention tree 0 is the node's own exact tree and trees
 * 1..P-1 are its read-only estimates of the peers' trees (Section 2: one trie per node plus N-1 peer
 * estimates).  Requests are routed in batches: every request is matched against every tree
 * (PrefixMatch of Algorithm 1) and sent to the argmax (getBestNode), with a load term.  Trees are
 * refreshed by anti-entropy: a full snapshot replaces a replica (Section 2, sendTrie; Section 3,
 * "Trie-broadcast loss"), or an ordered INSERT/DELETE delta patches it on the device (updateTrie /
 * updateTrieEstimate of Section 2 for INSERT; removal of a stored sequence for DELETE).
 *
 * Conventions
 *   - Tokens are int32 (any value).  A tree stores a multiset S(T) of token sequences.
 *   - match(r, T) = max over s in S(T) of LCP(r, s), 0 for an empty tree; this is the number of tokens
 *     of r found along one path of T, a partially matched edge included.
 *   - Route: score_p = match_p - alpha * load_p (exact, 64-bit); the chosen peer has the highest score,
 *     ties go to the lower load, then to the lower tree index.  Requires alpha >= 0, 0 <= load <= 65535,
 *     alpha * load <= 2^31 - 1 and P <= 65536.
 *   - Every call returns P2P_OK (0) or a negative error code; p2p_last_error() gives a message.  A call
 *     that fails leaves the router's trees unchanged, with one exception: p2p_tree_apply_delta_static,
 *     which may not grow a tree, returns P2P_E_NOMEM with the trees that ran out of room holding part of
 *     their ops (each op applied whole or not at all).
 *   - Device work is enqueued on the router's stream (p2p_router_set_stream); calls that take device
 *     pointers return before the work finishes.  Asynchronous device-side errors are reported by the
 *     next p2p_router_sync() as P2P_E_DEVICE.
 *   - The caller owns every buffer it passes; the library never frees caller memory.  Objects the
 *     library returns (routers, snapshots) are freed with their destroy/free call.
 *   - One router is used by one host thread at a time (the single writer of Section 3, "Asynchrony").
 */
#ifndef P2P_ROUTER_H
#define P2P_ROUTER_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
  P2P_OK = 0,
  P2P_E_INVAL = -1,   /* bad argument */
  P2P_E_NOMEM = -2,   /* allocation failed, or a tree outgrew the int32 flat format */
  P2P_E_FORMAT = -3,  /* malformed snapshot */
  P2P_E_CUDA = -4,    /* a CUDA runtime call failed */
  P2P_E_DEVICE = -5   /* a kernel reported an error (bad request offsets, internal consistency) */
};

enum { P2P_OP_INSERT = 0, P2P_OP_DELETE = 1 };
enum { P2P_KERNEL_COUNT = 27 }; /* kernels the kernel clock keeps totals for */
enum { P2P_MEM_HOST = 0, P2P_MEM_DEVICE = 1 };

typedef struct p2p_router p2p_router;
typedef struct p2p_snapshot p2p_snapshot;

/*
 * Flat radix tree: the full-snapshot wire format (Section 2, sendTrie).  n_nodes >= 1; node 0 is the root.
 *   label_off[v], label_len[v]  edge label of node v = labels[label_off[v] .. +label_len[v]); root: len 0,
 *                               every other node: len >= 1
 *   child_begin[v], child_count[v]  v's children are entries child_begin[v] .. +child_count[v] of
 *                               child_first_tok[] / child_idx[] (n_nodes - 1 entries in total)
 *   term_count[v]               number of stored sequences ending at v (>= 0)
 *   child_first_tok[e]          first label token of node child_idx[e]; strictly ascending within a node
 * Valid: every non-root node is listed exactly once as a child and is reachable from the root, every
 * non-root leaf and every non-root node with one child has term_count > 0, and every root-to-node path
 * has at most 2^31 - 1 tokens.  Canonical (as built and downloaded by the library): nodes in preorder,
 * children ascending, labels and child lists packed in node order.
 */
typedef struct p2p_flat_tree {
  int32_t n_nodes;
  int32_t n_labels;
  const int32_t* label_off;
  const int32_t* label_len;
  const int32_t* child_begin;
  const int32_t* child_count;
  const int32_t* term_count;
  const int32_t* child_first_tok;
  const int32_t* child_idx;
  const int32_t* labels;
} p2p_flat_tree;

/*
 * Segmented sequence list: sequence i is the concatenation of the pool runs
 * pool[seg_off[s] .. seg_off[s] + seg_len[s]) for s in [seg_begin[i], seg_begin[i+1]).  seg_begin has
 * n + 1 entries, non-decreasing, starting at 0 and ending at n_segs; every run lies inside the pool.
 * Runs may overlap, so a shared prefix is sent once and referenced by many sequences.
 */
typedef struct p2p_seqs {
  int64_t n;
  const int64_t* seg_begin;
  const int64_t* seg_off;
  const int32_t* seg_len;
  const int32_t* pool;
  int64_t n_segs;
  int64_t n_pool;
} p2p_seqs;

/*
 * Ordered anti-entropy delta: op[i] (P2P_OP_INSERT / P2P_OP_DELETE) applies to sequence i of seqs.
 * With peer = -1, peer_begin[P+1] (non-decreasing, from 0 to seqs.n) gives tree p the ops
 * peer_begin[p] .. peer_begin[p+1]-1; otherwise peer_begin is ignored and all ops go to one tree.
 * mem = P2P_MEM_HOST: every array is in host memory; P2P_MEM_DEVICE: every array is in device memory.
 */
typedef struct p2p_delta {
  const int32_t* op;
  p2p_seqs seqs;
  const int64_t* peer_begin;
  int32_t mem;
} p2p_delta;

/* ---- router ---------------------------------------------------------------------------------------- */

/* Creates a router with P >= 1 empty trees on the current CUDA device (Section 2: N-1 estimates plus the
 * own tree; a restarted node starts with empty trees, Section 2 crash-recovery model).  *out receives the
 * handle.  Errors: P2P_E_INVAL (P out of range, out NULL), P2P_E_CUDA, P2P_E_NOMEM. */
int p2p_router_create(int32_t P, p2p_router** out);

/* Frees the router and all device memory it owns (after finishing its queued work).  NULL is a no-op. */
void p2p_router_destroy(p2p_router* r);

/* Sets the CUDA stream (a cudaStream_t, NULL = legacy default stream) on which the router enqueues its
 * work; the previous stream is synchronized first, so no router work is left on it. */
int p2p_router_set_stream(p2p_router* r, void* stream);

/* Waits for the router's queued work and reports device-side errors raised since the last sync
 * (P2P_E_DEVICE, message in p2p_last_error; the error state is then cleared). */
int p2p_router_sync(p2p_router* r);

/* Message of the last failed call on r (or of the last failed p2p_router_create when r is NULL). */
const char* p2p_last_error(const p2p_router* r);

int32_t p2p_router_num_trees(const p2p_router* r);

/* Number of CUDA kernels the router has launched since creation (route, delta, bookkeeping kernels);
 * lets a caller count the device work a region of code issued.  Not part of the paper's method. */
int64_t p2p_router_launch_count(const p2p_router* r);

/* Kernel clock, a measurement aid (not part of the paper's method).  With on != 0 the router records a CUDA
 * event pair on its stream around each of its kernel launches and sums the device time per kernel; the
 * totals start from zero.  on = 0 switches the clock off and drops the totals.  Waits for queued work.
 * Each pair adds an event record before and after the launch, a few microseconds of stream work. */
int p2p_router_kernel_clock(p2p_router* r, int32_t on);

/* Totals of kernel i (0 <= i < P2P_KERNEL_COUNT, an index into the library's list of kernels) since the clock was
 * switched on: *name (nullable) receives the kernel's name (a static string), *launches and *ms (nullable)
 * the timed launches and their summed device time in milliseconds; 0 and 0.0 while the clock is off.
 * Waits for queued work.  Errors: P2P_E_INVAL (i out of range), P2P_E_CUDA. */
int p2p_router_kernel_time(p2p_router* r, int32_t i, const char** name, int64_t* launches, double* ms);

/* ---- snapshots (host only; no GPU needed) ---------------------------------------------------------- */

/* Builds the canonical snapshot of the multiset `seqs` (host pointers), i.e. the radix tree a node would
 * broadcast for these cached sequences (Section 2, sendTrie).  Errors: P2P_E_INVAL (malformed list),
 * P2P_E_NOMEM (tree beyond the int32 flat format). */
int p2p_snapshot_build(const p2p_seqs* seqs, p2p_snapshot** out);

/* Read-only view of a snapshot's arrays (valid until p2p_snapshot_free). */
void p2p_snapshot_view(const p2p_snapshot* s, p2p_flat_tree* out);

void p2p_snapshot_free(p2p_snapshot* s);

/* Checks a flat tree (host pointers) against the validity rules above: P2P_OK or P2P_E_FORMAT. */
int p2p_flat_tree_validate(const p2p_flat_tree* t);

/* ---- trees ----------------------------------------------------------------------------------------- */

/* Replaces tree `peer` with the full snapshot t (host pointers, copied before return).  This is the
 * receive side of the anti-entropy broadcast: delivering the same snapshot twice gives the same tree
 * (Section 3, "Trie-broadcast loss").  Enqueued on the router stream after earlier routes.
 * Device memory: the tree's arrays with headroom for deltas, plus a spare set a quarter larger that a
 * later device compaction copies the tree into (the old set then becomes the spare); the spare is skipped
 * when there is no room for it.
 * Errors: P2P_E_INVAL (peer), P2P_E_FORMAT (invalid tree; nothing changes), P2P_E_NOMEM, P2P_E_CUDA. */
int p2p_tree_upload(p2p_router* r, int32_t peer, const p2p_flat_tree* t);

/* Builds the canonical snapshot of `seqs` (host pointers) and uploads it as tree `peer`. */
int p2p_tree_build(p2p_router* r, int32_t peer, const p2p_seqs* seqs);

/* Exports tree `peer` as its canonical snapshot (waits for queued work).  Two trees holding the same
 * multiset export identical arrays.  *out is freed with p2p_snapshot_free. */
int p2p_tree_download(p2p_router* r, int32_t peer, p2p_snapshot** out);

/* Applies the ordered delta d to tree `peer` (0 <= peer < P), or, with peer = -1, to every tree p its
 * ops peer_begin[p] .. peer_begin[p+1]-1.  INSERT adds one occurrence of the sequence (Section 2,
 * updateTrie / updateTrieEstimate); DELETE removes one occurrence, and is a counted no-op when the
 * sequence is not stored.  Trees stay edge-compressed and canonical.  Runs on the device; the call
 * returns when the delta is applied (device arrays are only read, host arrays are copied).  A tree whose
 * stale arena space has passed its live space is then compacted on the device, and with it every tree of
 * the call at least 70% of the way there.
 * *n_absent (nullable) receives the number of no-op DELETEs.
 * Errors: P2P_E_INVAL (bad op code, peer, ranges or segments; nothing changes), P2P_E_NOMEM,
 * P2P_E_CUDA, P2P_E_DEVICE. */
int p2p_tree_apply_delta(p2p_router* r, int32_t peer, const p2p_delta* d, int64_t* n_absent);

/* As p2p_tree_apply_delta, for callers that cannot allocate memory while they patch replicas: a serving
 * loop whose device memory belongs to another allocator (it may not call cudaMalloc, cudaFree or a
 * caching allocator on its hot path), or a process whose device footprint must stay fixed after start-up.
 * The paper has no counterpart; this is a deployment variant of the delta call.
 * It allocates nothing, host or device: d must be in device memory (d->mem = P2P_MEM_DEVICE, else
 * P2P_E_INVAL); the delta is validated on the device; the call's scratch lives in one static device
 * array of the library (8 MiB plus a 256-byte header, held by every GPU that loads the library until the
 * process exits); trees are never grown or compacted.
 * Limits: the scratch holds one byte per op of the delta (rounded up to whole 4-byte words), plus, only
 * when some op's sequence is split into more than two pool runs, 64 bytes x (longest sequence in tokens)
 * per tree the call touches; a delta that needs more gets P2P_E_INVAL.  If a tree's arenas run out of room, the call returns P2P_E_NOMEM and that
 * tree holds only part of its ops (each op applied whole or not at all); p2p_tree_apply_delta, which may
 * allocate, grows trees.
 * Every call looks up the static array's device address (cudaGetSymbolAddress, with the router's device
 * current; the lookup allocates nothing).  The first lookup on a device may load the library's module
 * there, so make the first call before any stream capture.  Every
 * call shares the array, so calls whose device work overlaps (for example two routers on different
 * streams) race: order them.  The call returns when the delta is applied.  Other errors as
 * p2p_tree_apply_delta. */
int p2p_tree_apply_delta_static(p2p_router* r, int32_t peer, const p2p_delta* d, int64_t* n_absent);

/* Own-tree and estimate maintenance after routing (Algorithm 1): once request r has been sent to node k and
 * acknowledged, the sender inserts r into its estimate of k's trie (UpdateTrieEstimate(r, k)); a request the
 * node serves itself, k = its own tree (index 0 by convention), goes into its own trie (UpdateTrie; the
 * request's tokens stand in for the result, whose generated tokens are not known here).  For a routed batch:
 * request b is inserted once into tree peer[b]; requests with peer[b] < 0 (no route) are skipped.
 *   tokens      DEVICE int32[n_tokens]; request b is tokens[offsets[b] .. offsets[b+1]) (read, never copied)
 *   offsets     DEVICE int64[B+1]
 *   peer        DEVICE int32[B], as p2p_route_batch writes it (any values < P)
 *   n_inserted  (nullable) receives the number of requests inserted
 * The batch is counting-sorted by tree on the device into an INSERT delta held in router buffers and applied
 * like p2p_tree_apply_delta (arena growth and compaction included); inserts commute, so the trees equal those
 * of inserting the requests one by one in batch order.  Waits for the work.  B = 0 is a no-op; B <= 2^30.
 * Errors: P2P_E_INVAL (a peer >= P, or a routed request with offsets outside [0, n_tokens] or decreasing:
 * nothing changes), P2P_E_NOMEM, P2P_E_CUDA, P2P_E_DEVICE. */
int p2p_update_estimates(p2p_router* r, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets, int64_t B,
                         const int32_t* peer, int64_t* n_inserted);

/* ---- LRU cache trie (EvictLRUTrie of Algorithm 1) --------------------------------------------------------
 *
 * A node's own trie is its KV cache: Algorithm 1 inserts what the node serves (UpdateTrie) and, while a
 * request needs more memory than is free, evicts the least recently used leaf token, one token at a time
 * (Section 2 primitive list: evictLRUTrie).  A tree made an LRU tree keeps a last-access time per token
 * (stored per node: an access that ends inside an edge splits the edge there, so every edge's tokens share
 * one time).  Times are caller-given integers that never decrease, at most 2^32 - 2.  Semantics, per token:
 *   - an insert at time t touches every token of the sequence's path; an access at time t touches the
 *     request's matched tokens;
 *   - an eviction removes the leaf token with the oldest last access, ties to the lexicographically smallest
 *     token path (signed token order); sequences that ended at it now end one token earlier.
 * An LRU tree changes only through these calls: uploads, deltas and p2p_update_estimates that would change it
 * are rejected (P2P_E_INVAL).  It is routed like any tree, and its export is canonical.  It is not compacted
 * (evicted nodes stay in its arenas as stale space).
 */

/* Makes tree `tree` an LRU tree; its current tokens get time 0.  A no-op if it is one already. */
int p2p_lru_enable(p2p_router* r, int32_t tree);

/* UpdateTrie of a batch at time `time`: each request (DEVICE tokens/offsets as for p2p_route_batch) is
 * inserted once, then every token of its path is touched.  Waits for the work.  Errors: P2P_E_INVAL (not an
 * LRU tree, time out of order, invalid offsets: nothing changes), P2P_E_NOMEM, P2P_E_CUDA. */
int p2p_lru_insert(p2p_router* r, int32_t tree, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets,
                   int64_t B, int64_t time);

/* Requests served from the cache at time `time`: each request's matched tokens are touched, and
 * out_match (DEVICE int32[B], nullable) receives PrefixMatch(r_b, tree).  Waits for the work.  Requests with
 * invalid offsets match 0, touch nothing and make the next p2p_router_sync return P2P_E_DEVICE.  Errors:
 * P2P_E_INVAL, P2P_E_NOMEM (no room to split edges), P2P_E_CUDA. */
int p2p_lru_access(p2p_router* r, int32_t tree, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets,
                   int64_t B, int64_t time, int32_t* out_match);

/* EvictLRUTrie n_tokens times: removes the n_tokens least recently used leaf tokens in the order above (all
 * of them if the tree holds fewer); *n_evicted (nullable) receives how many.  The removal is done at once on
 * the device (the order is that of one-token evictions; see lru_kernel.cu).  Waits for the work.  Errors:
 * P2P_E_INVAL, P2P_E_CUDA, P2P_E_DEVICE. */
int p2p_lru_evict(p2p_router* r, int32_t tree, int64_t n_tokens, int64_t* n_evicted);

/* Section 5's expected cache hit rate of routed requests: out[b] = match[b*P + peer[b]] / |r_b| in single
 * precision (IEEE division, rounded to nearest), 0 for an empty request or peer[b] < 0.  match (DEVICE
 * int32[B*P]), offsets (DEVICE int64[B+1]), peer (DEVICE int32[B]) as p2p_route_batch writes and reads them;
 * out DEVICE float[B].  Asynchronous on the router stream.  Errors: P2P_E_INVAL. */
int p2p_hit_rate(p2p_router* r, const int32_t* match, const int64_t* offsets, int64_t B, const int32_t* peer,
                 float* out);

/* Sizes of tree `peer`: out[0] live nodes (root included), out[1] node slots in use, out[2] child
 * entries in use, out[3] label tokens in use, out[4] stale child entries, out[5] stale label tokens,
 * out[6..8] node / child-entry / label capacities.  Waits for queued work. */
int p2p_tree_stats(p2p_router* r, int32_t peer, int64_t out[9]);

/* ---- routing --------------------------------------------------------------------------------------- */

/* Routes a batch of B requests (Algorithm 1: k = argmax_j PrefixMatch(r, T_j), with the load term).
 *   tokens      DEVICE int32[n_tokens]; request b is tokens[offsets[b] .. offsets[b+1])
 *   offsets     DEVICE int64[B+1]; a request with 0 <= offsets[b] <= offsets[b+1] <= n_tokens violated
 *               gets match 0 and peer -1 and makes the next p2p_router_sync return P2P_E_DEVICE
 *   load        HOST int32[P], copied before return; alpha >= 0 (see Conventions)
 *   out_match   DEVICE int32[B*P], row-major: out_match[b*P + p] = match(r_b, T_p)
 *   out_peer    DEVICE int32[B]: the chosen tree of request b
 * Asynchronous on the router stream.  B = 0 is a no-op; B may be at most 2^30 (split larger batches).
 * Errors: P2P_E_INVAL, P2P_E_CUDA. */
int p2p_route_batch(p2p_router* r, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets, int64_t B,
                    const int32_t* load, int32_t alpha, int32_t* out_match, int32_t* out_peer);

/* p2p_route_batch with the route decision of p2p_route_decide made in the same pass: the walk kernels keep
 * the two largest route keys of the trees not excluded while they write the match row, so the match matrix
 * is not read again (Section 3.2, hot specialist push-back: no routing to a peer that pushed back; Section
 * 3.3, in-flight forwarded request failure: no routing to a suspected-failed peer, and the next-best target
 * for a forwarding timeout).
 *   excluded    HOST uint8[P] (nullable = none), copied before return: excluded[p] != 0 takes tree p out of
 *               the candidates (its match column is still written)
 *   out_peer    DEVICE int32[B]: the first candidate of the route order, -1 if every tree is excluded
 *   out_next    DEVICE int32[B] (nullable): the second candidate, -1 if there is none
 * Other arguments, limits and errors as p2p_route_batch; out_match is the same.  With excluded and out_next
 * both NULL this is p2p_route_batch.  Asynchronous on the router stream. */
int p2p_route_batch_decide(p2p_router* r, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets, int64_t B,
                           const int32_t* load, int32_t alpha, const uint8_t* excluded, int32_t* out_match,
                           int32_t* out_peer, int32_t* out_next);

/* Announces the next batch to route (DEVICE tokens/offsets as for p2p_route_batch; B <= 2^30).  The route's
 * first step, grouping requests by shared prefix, reads only the requests, so the next p2p_tree_apply_delta
 * launches it on a low-priority side stream right after its delta kernel: it runs on the SM room the delta
 * kernel leaves.  The next p2p_route_batch or p2p_route_batch_decide of the same batch (same pointers and
 * sizes) waits for it instead of grouping; a route of another batch groups as usual.  The requests must not
 * change between the two calls.  Not part of the paper's method: a scheduling aid for a step of delta +
 * route.  Errors: P2P_E_INVAL. */
int p2p_route_prepare(p2p_router* r, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets, int64_t B);

/* As p2p_route_batch with every pointer in HOST memory: copies the requests to the device, routes,
 * copies both outputs back and waits.  Large batches go in up to 8 chunks of at least 131,072 requests:
 * a chunk's inputs are copied in while the chunk before it is routed and the one before that is copied
 * out (two copy streams of the router, ordered by events against the router stream).  Results equal
 * those of one p2p_route_batch of the whole batch.  The copies overlap only from pinned host memory.
 * Offsets are validated on the host (P2P_E_INVAL).  Requests are tokens[offsets[0] .. offsets[B]). */
int p2p_route_batch_host(p2p_router* r, const int32_t* tokens, const int64_t* offsets, int64_t B,
                         const int32_t* load, int32_t alpha, int32_t* out_match, int32_t* out_peer);

/* Route decision with excluded peers and a fallback target, from a batch's match matrix.  Section 3.2
 * (hot specialist push-back) stops routing to a peer that advertised back-pressure; Section 3.3
 * (in-flight forwarded request failure) marks a peer that missed its broadcasts as suspected-failed, and on
 * a forwarding timeout sends the request to the next-best target, which may be the node itself.
 *   match       DEVICE int32[B*P] row-major, as p2p_route_batch writes it (values below 0 count as 0)
 *   load        HOST int32[P], alpha: as for p2p_route_batch; copied before return
 *   excluded    HOST uint8[P] (nullable = none): excluded[p] != 0 takes tree p out of the candidates;
 *               copied before return
 *   out_peer    DEVICE int32[B]: the first candidate of the route order (match - alpha*load, then the lower
 *               load, then the lower index), -1 if every tree is excluded
 *   out_next    DEVICE int32[B]: the second candidate of that order, -1 if there is none
 * With nothing excluded, out_peer equals p2p_route_batch's out_peer.  Asynchronous on the router stream;
 * one kernel launch.  B = 0 is a no-op.  Errors: P2P_E_INVAL (B < 0, NULL pointers, load or alpha out of
 * range), P2P_E_CUDA. */
int p2p_route_decide(p2p_router* r, const int32_t* match, int64_t B, const int32_t* load, int32_t alpha,
                     const uint8_t* excluded, int32_t* out_peer, int32_t* out_next);

#ifdef __cplusplus
}
#endif
#endif /* P2P_ROUTER_H */
