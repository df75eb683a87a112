// internal.h -- device layout of the trees and the kernel launchers shared by the library's sources.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <cstring>
#include <string>
#include <vector>

#include "p2p_router.h"

// Host snapshot object handed out by p2p_snapshot_build / p2p_tree_download (layout of p2p_flat_tree).
struct p2p_snapshot {
  int32_t n_nodes = 0, n_labels = 0;
  std::vector<int32_t> label_off, label_len, child_begin, child_count, term_count, child_first_tok, child_idx, labels;
};

namespace p2p {

// Device layout of one tree (HBM, one allocation per array):
//   node[v]  = {tab_off, meta, live, term_count}                          (int4, 16 B)
//              v's children live in an open-addressing hash table of 2^(meta & 31) slots at
//              child[tab_off ..] (no table when meta == 0); meta >> 5 counts the slots ever claimed
//              (live children + tombstones); live = number of children; term_count = sequences ending at v.
//   child[s] = {first_tok, node, label_off, label_len}: one slot of a children table (int4, 16 B).
//              .node: 0 = empty slot (the slot is all zero), >= 1 = the child, -1 = removed (tombstone,
//              key kept), -3 = being claimed during a delta.  Slots are probed linearly from a
//              multiplicative hash of first_tok.
//   label[]  = int32 tokens of the tree's own label arena.  An edge's label is label[label_off ..
//              +label_len) when label_off >= 0, and shared[~label_off ..] when label_off < 0: long labels
//              are interned in a router-wide pool (the same few-shot prefixes are cached by many peers, so
//              one copy serves every replica that holds it).
// Node 0 is the root.  Keeping the child's label position in its slot lets a walk start comparing the
// label as soon as the lookup returns; every lookup is one coalesced probe of 32 consecutive slots.
struct TreeView {
  const int4* node;
  const int4* child;
  const int32_t* label;
  const int32_t* shared;        // the router's shared label pool
  const uint32_t* rfilter;      // the root's first-token filter (see below)
  int32_t root_off, root_bits;  // the root's children table (copied from node[0] when the view is set)
};

// Root first-token filter, one per tree: a bit per 16-bit hash of a token, set for the first token of every
// child the root has had since the tree was uploaded (bits are never cleared, so a clear bit proves the token
// starts no child; a set bit may be stale).  A request whose first token is absent matches nothing in the
// tree; the filter (8 KB a tree, 2 MB for 256 trees) stays in L2, while the root tables it spares (~1 MB a
// tree at the scale workload) do not.  Fresh prompts, a fifth of the scale workload's requests, are such
// requests in most trees.
constexpr int kRootFilterWords = 2048;
inline __host__ __device__ uint32_t root_filter_bit(int32_t tok) { return ((uint32_t)tok * 0xC2B2AE3Du) >> 16; }
inline __host__ __device__ bool root_filter_has(const uint32_t* f, int32_t tok) {
  const uint32_t h = root_filter_bit(tok);
  return (f[h >> 5] >> (h & 31)) & 1u;
}

// Start of the label of an edge whose label_off is `off` (see the layout above).
inline __host__ __device__ const int32_t* label_ptr(const int32_t* label, const int32_t* shared, int32_t off) {
  return off >= 0 ? label + off : shared + ~off;
}
// label_off of the same label advanced by k tokens.
inline __host__ __device__ int32_t label_adv(int32_t off, int32_t k) { return off >= 0 ? off + k : off - k; }

// Mutable state of one tree, shared by the delta kernel's warps for that tree (counters updated with
// atomics) and mirrored on the host between calls.
struct TreeState {
  int4* node;
  int4* child;
  int32_t* label;
  uint32_t* rfilter;           // the root's first-token filter (kRootFilterWords words; the router's array)
  uint32_t* stamp;             // LRU trees only (else NULL): per node slot, the last access of its edge's tokens
  int32_t n_node, cap_node;    // node slots used (bump arena) / capacity
  int32_t n_child, cap_child;  // child-table slots used (bump arena) / capacity
  int32_t n_label, cap_label;  // label tokens used (bump arena) / capacity
  int32_t status;              // DELTA_* bits
  int32_t need_node, need_child, need_label, need_root;  // largest request that did not fit
  int32_t pad_;
  int64_t op_begin, op_end;    // this call's ops for the tree: [op_begin, op_end)
  int64_t n_absent;            // DELETEs of sequences that were not stored
  int64_t stale_child, stale_label, dead_nodes;  // unreachable arena space
};

enum { DELTA_OK = 0, DELTA_NEED_SPACE = 1, DELTA_CORRUPT = 2 };

// Delta kernel: ops are bucketed by a hash of their first token (kDeltaBuckets per tree); one CTA of
// kDeltaWarps warps per tree takes the buckets heaviest first.
constexpr int kDeltaBucketBits = 5;
constexpr int kDeltaBuckets = 1 << kDeltaBucketBits;
constexpr int kDeltaWarps = 16;

// Children tables: at least 4 slots; grown when claimed slots (live and tombstoned) would pass 1/2 of the
// table, to at most 1/4 live load.  A lookup of a missing child, the common case for a request that leaves
// the cached prefixes, then scans about two slots of the linear probe.
constexpr int kMinTabBits = 2;
inline __host__ __device__ int32_t tab_bits(int32_t meta) { return meta & 31; }
inline __host__ __device__ int32_t tab_used(int32_t meta) { return (int32_t)((uint32_t)meta >> 5); }
inline __host__ __device__ int32_t make_meta(int32_t bits, int32_t used) { return bits | (int32_t)((uint32_t)used << 5); }
inline __host__ __device__ bool tab_full(int32_t bits, int64_t used_after) {
  return bits == 0 || used_after * 2 > ((int64_t)1 << bits);
}
constexpr int32_t kMaxTabBits = 26;  // slots ever claimed must fit the 27 bits of meta

// Kernel clock: per-kernel device time of a router's launches, a measurement aid (not part of the method).
// Launchers bracket every launch with clock_mark(id, ...); a router whose clock is on installs it in
// t_clock for the duration of an API call on the calling thread (one router per host thread at a time).
enum KernelId {
  K_GROUP_HASH, K_GROUP_RESOLVE, K_GROUP_RESOLVE32, K_ROUTE_STAGED, K_LANE_LEADER, K_LANE_FOLLOWER, K_DECIDE,
  K_VALIDATE, K_INIT_RANGES, K_DELTA, K_COMPACT, K_COMPACT_LABELS, K_REFRESH_VIEWS, K_SET_TREE,
  K_UPDATE_COUNT, K_UPDATE_SCAN, K_UPDATE_SCATTER, K_GROUP_RANGES, K_GROUP_PLACE, K_LRU_WALK, K_LRU_STAMP,
  K_LRU_ORDER, K_LRU_SELECT, K_LRU_EVICT, K_LRU_OPS, K_HIT_RATE, K_ROOM, K_COUNT_
};
static_assert((int)K_COUNT_ == (int)P2P_KERNEL_COUNT, "the header's kernel count");
const char* kernel_name(int id);
struct KernelClock {
  virtual void mark(int id, bool end, cudaStream_t st) = 0;
  virtual ~KernelClock() = default;
};
extern thread_local KernelClock* t_clock;
inline void clock_mark(int id, bool end, cudaStream_t st) {
  if (t_clock) t_clock->mark(id, end, st);
}
// One timed launch: the variadic part is the kernel<<<...>>>(...) expression.
#define P2P_TIMED(id, st, ...)          \
  do {                                  \
    ::p2p::clock_mark(id, false, st);   \
    __VA_ARGS__;                        \
    ::p2p::clock_mark(id, true, st);    \
  } while (0)

// Bits of the router's device error word.
enum { ERR_BAD_OFFSETS = 1, ERR_CORRUPT_TREE = 2, ERR_STALL = 4 };

// Shared-prefix groups of a batch (group_kernel.cu): requests of at least kGroupHead tokens are grouped by
// their first kGroupHead tokens; lead[b] is b's group leader, cpre[b] its exact common prefix with the
// leader (followers only); lists[0 .. counts[0]) are the leaders, lists[B .. B + counts[1]) the followers,
// each group's followers side by side (so the warps routing them at the same time share the leader's row,
// checkpoints and tables in cache).
constexpr int kGroupHead = 64;
struct GroupScratch {
  unsigned long long* keys;  // 2^bits slots
  int32_t* vals;             // 2^bits slots
  int32_t bits;
  int32_t* slot_of;  // [B]
  int32_t* lead;     // [B]
  int32_t* cpre;     // [B]
  int32_t* lists;    // [2B]
  int32_t* counts;   // [8]: leaders, followers, groups with a checkpoint row, the leader pass's work cursor,
                     //      the follower ranges handed out
  int32_t* fcnt;     // [B]: a leader's follower count, then the start of its followers' range
  int32_t* gid;      // [B]: a leader's checkpoint row (-1: none)
  int32_t* cmin;     // [B]: a leader's smallest common prefix with its followers
  int4* ckpt;        // [gcap * P]: per (row, tree) the leader's walk state to resume from (see route_kernel.cu)
  int32_t gcap;      // checkpoint rows
};
cudaError_t launch_group(const int32_t* tokens, int64_t n_tokens, int64_t tok_base, const int64_t* offsets, int64_t B,
                         const GroupScratch& g, int num_sms, cudaStream_t st);

// Staged load words (d_load) carry the load in the low 16 bits and kLoadExcluded for a tree that the
// decision with excluded trees takes out.
constexpr int32_t kLoadExcluded = 1 << 16;
// Best and next-best non-excluded peer of every row of match [B x P] (route_key order); -1 where none.
cudaError_t launch_decide(const int32_t* match, int64_t B, int32_t P, const int32_t* d_load, int32_t alpha,
                          int32_t* out_peer, int32_t* out_next, int num_sms, cudaStream_t st);
// Route kernels (lookup + route decision) of a grouped batch, see route_kernel.cu: a leader pass and a
// follower pass (g is required).  *launched is set to the number of kernels launched.  With decide (load
// words carrying kLoadExcluded) or out_next (device [B]) the passes make the decision with excluded trees
// and the next-best target instead of the plain argmax.
cudaError_t launch_route(const TreeView* d_trees, int32_t P, const int32_t* tokens, int64_t n_tokens,
                         int64_t tok_base, const int64_t* offsets, int64_t B, const int32_t* d_load, int32_t alpha,
                         int32_t* out_match, int32_t* out_peer, int32_t* d_err, const GroupScratch* g, int num_sms,
                         cudaStream_t st, int* launched, bool decide = false, int32_t* out_next = nullptr);

// Delta kernel: applies the ops [op_begin, op_end) of states[0 .. n_trees), one CTA of kDeltaWarps warps
// per tree, or per part of a tree: with parts (n_blocks words, one per CTA: tree | part << kPartShift |
// nparts << kNpartShift) a tree's ops are split among nparts CTAs by first-token bucket modulo nparts
// (1 <= nparts <= kDeltaBuckets).  done[i] (one byte per op of the call, zero before the first launch, kept
// across relaunches) marks the ops applied so far.  gather (CTAs * kDeltaWarps * gather_stride tokens) is
// needed only when an op's sequence has more than two pool runs; otherwise it may be NULL.
// A launch-wide table of verified (interned label, pool run) equalities (keys all zero before a call's first
// launch; keys [mask + 1], vals [mask + 1]).  NULL: none (the allocation-free call).
struct GlobalMemo {
  unsigned long long* keys;
  int32_t* vals;
  uint32_t mask;
};
constexpr int kGlobalMemoBits = 16;
cudaError_t launch_delta(TreeState* d_states, uint8_t* done, int32_t n_trees, const int32_t* op,
                         const int64_t* seg_begin, const int64_t* seg_off, const int32_t* seg_len, const int32_t* pool,
                         int32_t* gather, int64_t gather_stride, const int32_t* shared, cudaStream_t st,
                         const GlobalMemo* gm = nullptr, const int32_t* parts = nullptr, int32_t n_blocks = 0);
constexpr int kPartShift = 16, kNpartShift = 21;
constexpr int32_t kPartTreeMask = (1 << kPartShift) - 1;  // a tree index < 65,536 (P <= 65,536)
static_assert(kDeltaBuckets <= 32, "a part index fits in 5 bits and nparts in 6");

// Compaction: copies the live part of a tree (everything reachable from the root) into fresh arrays, with
// nodes renumbered in breadth-first order, every live table rehashed at its size without tombstones, and
// own-arena labels packed (shared-pool labels stay where they are).  One CTA per job.
struct CompactJob {
  const int4* node;  // old arrays
  const int4* child;
  const int32_t* label;
  int4* nnode;  // new arrays and their capacities
  int4* nchild;
  int32_t* nlabel;
  int4* queue;  // cap_node entries of scratch, by new id: (old id, old label offset, new label offset,
                //   own-arena label length or 0)
  int32_t cap_node, cap_child, cap_label;
  int32_t n_node, n_child, n_label;  // out: the new counts
  int32_t status;                    // out: 0, or 1 if a new array was too small (the job is then void)
  int32_t pad_;
};
// Two launches: compact_kernel (one CTA per job) copies the structure, then compact_labels_kernel moves the
// labels of every job over the whole GPU.  max_cap_node bounds every job's cap_node.
cudaError_t launch_compact(CompactJob* d_jobs, int32_t n_jobs, int32_t max_cap_node, int num_sms, cudaStream_t st);

// Home slot of a first token in a children table of 2^bits slots (host table builder and kernels).
inline __host__ __device__ uint32_t slot_hash(int32_t tok, int32_t bits) {
  return bits ? ((uint32_t)tok * 0x9E3779B1u) >> (32 - bits) : 0u;
}

// Writes a tree's state and view on the device (values passed as kernel parameters, so no host buffer
// has to outlive the call).
cudaError_t launch_set_tree(TreeState* d_state, TreeView* d_view, TreeState value, const int32_t* shared,
                            cudaStream_t st);

// Rewrites views[0 .. n) from states[0 .. n) (after a delta moved some trees' arrays).
cudaError_t launch_refresh_views(const TreeState* d_states, TreeView* d_views, int32_t n, const int32_t* shared,
                                 cudaStream_t st);

// Static scratch of the allocation-free delta call (delta_static.cu).
enum { STATIC_BAD_OP = 1, STATIC_BAD_SEGMENT = 2, STATIC_BAD_PEER_BEGIN = 4, STATIC_TOO_LONG = 8 };
int64_t static_scratch_tokens();
cudaError_t static_scratch(int device, int32_t** header, int32_t** tokens);
// Validates a device-resident delta on the device into a kStaticHeaderInts-word header (zeroed first):
// [0..1] longest sequence (u64), [2] STATIC_* error bits, [3] most pool runs of one op.
cudaError_t launch_validate(int32_t* header, const p2p_delta* d, int32_t peer, int32_t P, cudaStream_t st);
cudaError_t launch_init_ranges(TreeState* d_states, int32_t nt, const int64_t* peer_begin, int64_t n, cudaStream_t st);
// Per tree that stopped for room (DELTA_NEED_SPACE): room[2i] = label tokens and room[2i + 1] = INSERTs of its ops
// not yet applied (upper bounds of the room the rest of the call takes).
cudaError_t launch_room(const TreeState* d_states, int32_t nt, const uint8_t* done, const int32_t* op,
                        const int64_t* seg_begin, const int32_t* seg_len, long long* room, cudaStream_t st);
constexpr int kStaticHeaderInts = 64;

// A routed batch as a device-resident INSERT delta (update_kernel.cu).  counts [P] must be zero and bad [1]
// zero before the count launch; bad receives 1 (a peer >= P) | 2 (a routed request with invalid offsets).
// The scan writes peer_begin [P+1], the scatter cursors [P], seg_begin[n] = n and *total = n; the scatter
// fills op, seg_begin, seg_off and seg_len [n] (each op one run of the request's tokens).
cudaError_t launch_update_count(const int32_t* peer, const int64_t* offsets, int64_t B, int64_t n_tokens, int32_t P,
                                int32_t* counts, int32_t* bad, int num_sms, cudaStream_t st);
cudaError_t launch_update_scan(const int32_t* counts, int32_t P, int64_t* peer_begin, int32_t* cursor,
                               int64_t* seg_begin_end, int64_t* total, cudaStream_t st);
cudaError_t launch_update_scatter(const int32_t* peer, const int64_t* offsets, int64_t B, int64_t n_tokens, int32_t P,
                                  int32_t* cursor, int32_t* op, int64_t* seg_begin, int64_t* seg_off, int32_t* seg_len,
                                  int num_sms, cudaStream_t st);

// LRU trees (lru_kernel.cu): walk + stamp (an access), BFS order, the level passes, the selection counts and
// the eviction; see that file for the method.  lvl_begin (host) holds n_levels + 1 offsets into order.
cudaError_t launch_lru_walk(const TreeState& s, const int32_t* shared, const int32_t* tokens, int64_t n_tokens,
                            const int64_t* offsets, int64_t B, int32_t* touch, int32_t* pslot, int32_t* out_match,
                            int32_t* err, int num_sms, cudaStream_t st);
cudaError_t launch_lru_stamp(const TreeState& s, TreeState* d_state, const int32_t* shared, const int32_t* touch,
                             const int32_t* pslot, int32_t n_node, uint32_t time, int num_sms, cudaStream_t st);
cudaError_t launch_lru_bfs(const TreeState& s, const int32_t* front, int32_t n_front, int32_t* next, int32_t* n_next,
                           int32_t cap, int32_t* parent, int32_t* cslot, int num_sms, cudaStream_t st);
cudaError_t launch_lru_init(const int32_t* order, int32_t n, int64_t* size, int64_t* off, int64_t* rank,
                            unsigned long long* best, uint8_t* gone, int num_sms, cudaStream_t st);
// Scratch of the sibling-offset sort (n2 = the live non-root nodes rounded up to a power of two; N = node slots).
struct LruSortScratch {
  unsigned long long* key;  // [n2]
  int32_t* val;             // [n2]
  int32_t* first;           // [N]
  int64_t* scan;            // [n2]
};
cudaError_t launch_lru_levels(const TreeState& s, const int32_t* order, const int32_t* lvl_begin, int32_t n_levels,
                              const int32_t* parent, const int32_t* cslot, int64_t* size, int64_t* off, int64_t* rank,
                              unsigned long long* best, int32_t* end, const LruSortScratch& sc, int num_sms,
                              cudaStream_t st);
cudaError_t launch_lru_count(const TreeState& s, const int32_t* nodes, int32_t n, const int32_t* cslot,
                             const int64_t* rank, const int32_t* end, int mode, uint32_t S, unsigned long long K,
                             unsigned long long* out, int num_sms, cudaStream_t st);
cudaError_t launch_lru_evict(const TreeState& s, TreeState* d_state, const int32_t* order, const int32_t* lvl_begin,
                             int32_t n_levels, const int32_t* parent, const int32_t* cslot, const int64_t* rank,
                             const int32_t* end, uint32_t S, unsigned long long K, int32_t cut, uint8_t* gone,
                             int32_t* surv, int num_sms, cudaStream_t st);
cudaError_t launch_lru_ops(const int64_t* offsets, int64_t B, int64_t n_tokens, int32_t* op, int64_t* seg_begin,
                           int64_t* seg_off, int32_t* seg_len, int num_sms, cudaStream_t st);
cudaError_t launch_hit_rate(const int32_t* match, int32_t P, const int64_t* offsets, int64_t B, const int32_t* peer,
                            float* out, int num_sms, cudaStream_t st);

// Host-side helpers in snapshot.cpp.
void set_global_error(const std::string& msg);
const char* global_error();
// Checks a segmented sequence list (ranges only; the pool is not read).  max_len / lens: optional outputs.
bool check_seqs(const p2p_seqs* s, std::string& err, int64_t* max_len, std::vector<int64_t>* lens);
bool build_snapshot(const p2p_seqs& S, p2p_snapshot& out, std::string& err);
bool validate_flat(const p2p_flat_tree* t, std::string& err);
bool snapshot_from_device_layout(const int4* node, int64_t n_node, const int4* child, int64_t n_child,
                                 const int32_t* label, int64_t n_label, const int32_t* shared, int64_t n_shared,
                                 p2p_snapshot& out, std::string& err);

}  // namespace p2p
