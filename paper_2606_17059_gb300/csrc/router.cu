// router.cu -- host runtime of the routing engine: the C ABI declared in p2p_router.h.
//
// The router owns P trees in HBM (layout in internal.h), allocated from a router-private stream-ordered
// memory pool so that replacing a tree (snapshot upload, arena growth) frees the old arrays in stream
// order, after any route still reading them.  Each tree also keeps a spare set of arrays that device
// compaction copies it into (the old set becomes the next spare).  All device work goes to the router's
// stream.
#include <algorithm>
#include <cstring>
#include <string>
#include <unordered_map>
#include <vector>

#include "internal.h"

using p2p::TreeState;
using p2p::TreeView;

namespace {

constexpr int kLoadRing = 8;
// p2p_route_batch_host pipelines its copies with the routing in up to kPipe chunks of at least
// kPipeRequests requests each.
constexpr int kPipe = 8;
constexpr int64_t kPipeRequests = 131072;
// Largest batch of one routing call: the grouping kernels and the pass lists index requests with int32.
constexpr int64_t kMaxBatch = (int64_t)1 << 30;

struct DevBuf {
  void* p = nullptr;
  size_t cap = 0;
};

int32_t clamp_i32(int64_t v) { return (int32_t)std::min<int64_t>(v, INT32_MAX); }

// Capacity of a tree's own label arena holding `own` live tokens.  Deltas leave replaced labels behind as
// stale space, and a tree is compacted once that passes its live space; twice the live tokens plus a
// quarter is enough to get there without growing the arena on the way.
int32_t label_cap(int64_t own) { return clamp_i32(2 * own + std::max<int64_t>(own / 4, 65536)); }

int64_t next_pow2(int64_t v) {
  int64_t p = 1;
  while (p < v) p <<= 1;
  return p;
}
int32_t log2_exact(int64_t p) {
  int32_t b = 0;
  while (((int64_t)1 << b) < p) ++b;
  return b;
}
// Labels at least this long are interned in the router's shared pool (shorter ones stay in the tree's
// own arena): the long runs are the shared prompt prefixes that many replicas hold.  Interned runs are also
// indexed by their first kHeadTokens tokens (a few per head), to find a run that a longer label starts with.
constexpr int32_t kInternMin = 128;
constexpr int32_t kHeadTokens = 64;
constexpr size_t kHeadCandidates = 8;

// 64-bit content hash of a token run (FNV-1a over the 32-bit tokens, then a final avalanche); interning
// always verifies the content, so a collision only means a run is not shared.
uint64_t run_hash(const int32_t* p, int64_t n) {
  uint64_t h = 0xcbf29ce484222325ull ^ (uint64_t)n;
  for (int64_t i = 0; i < n; ++i) h = (h ^ (uint32_t)p[i]) * 0x100000001b3ull;
  h ^= h >> 33;
  h *= 0xff51afd7ed558ccdull;
  return h ^ (h >> 33);
}

// Children-table sizes (log2 slots): load factor <= 1/4 at upload (tables grow past 1/2); the root's table
// gets extra room (at least 64 slots) because only the host can grow it.
int32_t table_bits_for(int64_t live, bool root) {
  if (root) return log2_exact(next_pow2(std::max<int64_t>(64, 4 * live + 64)));
  return live == 0 ? 0 : std::max<int32_t>(p2p::kMinTabBits, log2_exact(next_pow2(4 * live)));
}

// Inserts entry e into the table of 2^bits slots at tab (linear probing from its home slot).
void table_put(int4* tab, int32_t bits, const int4& e) {
  const uint32_t mask = (1u << bits) - 1;
  uint32_t s = p2p::slot_hash(e.x, bits);
  while (tab[s].y != 0) s = (s + 1) & mask;
  tab[s] = e;
}

}  // namespace

namespace p2p {

thread_local KernelClock* t_clock = nullptr;

const char* kernel_name(int id) {
  static const char* const names[K_COUNT_] = {
      "group_hash_kernel", "group_resolve_kernel", "group_resolve32_kernel", "route_kernel", "lane_kernel<true>",
      "lane_kernel<false>", "decide_kernel", "validate_kernel", "init_ranges_kernel", "delta_kernel",
      "compact_kernel", "compact_labels_kernel", "refresh_views_kernel", "set_tree_kernel", "update_count_kernel",
      "update_scan_kernel", "update_scatter_kernel", "group_ranges_kernel", "group_place_kernel", "lru_walk_kernel",
      "lru_stamp_kernel", "lru_order_kernels", "lru_count_kernel", "lru_evict_kernel", "lru_ops_kernel",
      "hit_rate_kernel", "room_kernel"};
  return id >= 0 && id < K_COUNT_ ? names[id] : "";
}

}  // namespace p2p

namespace {

// The router's kernel clock: an event pair recorded around each launch on the launch stream; the pairs are
// resolved into per-kernel totals when the totals are read (or when many are pending).
struct RouterClock final : p2p::KernelClock {
  struct Pending {
    int id;
    cudaEvent_t a, b;
  };
  std::vector<cudaEvent_t> spare;
  std::vector<Pending> pending;
  int open_id = -1;
  cudaEvent_t open_ev = nullptr;
  double ms[p2p::K_COUNT_] = {};
  int64_t n[p2p::K_COUNT_] = {};
  cudaError_t err = cudaSuccess;

  cudaEvent_t get() {
    if (!spare.empty()) {
      cudaEvent_t e = spare.back();
      spare.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) {
      err = cudaErrorMemoryAllocation;
      return nullptr;
    }
    return e;
  }
  void mark(int id, bool end, cudaStream_t st) override {
    if (!end) {
      open_id = id;
      open_ev = get();
      if (open_ev) cudaEventRecord(open_ev, st);
      return;
    }
    cudaEvent_t b = get();
    if (open_ev && b && open_id == id) {
      cudaEventRecord(b, st);
      pending.push_back(Pending{id, open_ev, b});
    } else {
      if (open_ev) spare.push_back(open_ev);
      if (b) spare.push_back(b);
    }
    open_ev = nullptr;
    open_id = -1;
    if (pending.size() >= 65536) resolve();
  }
  // Waits for the pending pairs and adds them to the totals.
  void resolve() {
    for (const Pending& q : pending) {
      float t = 0.f;
      if (cudaEventSynchronize(q.b) == cudaSuccess && cudaEventElapsedTime(&t, q.a, q.b) == cudaSuccess) {
        ms[q.id] += t;
        n[q.id] += 1;
      }
      spare.push_back(q.a);
      spare.push_back(q.b);
    }
    pending.clear();
  }
  void reset() {
    resolve();
    std::fill(ms, ms + p2p::K_COUNT_, 0.0);
    std::fill(n, n + p2p::K_COUNT_, 0);
  }
  ~RouterClock() override {
    resolve();
    for (cudaEvent_t e : spare) cudaEventDestroy(e);
  }
};

}  // namespace

struct p2p_router {
  int32_t P = 0;
  int device = 0;
  int num_sms = 0;
  cudaStream_t stream = nullptr;
  cudaMemPool_t pool = nullptr;
  std::vector<TreeState> hs;  // host mirror of every tree's state
  // Per tree, a second set of arrays (pointers and capacities) that a device compaction copies the tree
  // into; the old set then becomes the spare.  Empty when it could not be allocated.
  std::vector<TreeState> spare;
  TreeView* d_views = nullptr;
  TreeState* d_states = nullptr;
  uint32_t* d_rfilter = nullptr;  // P root first-token filters of kRootFilterWords words
  int32_t* d_load = nullptr;
  int32_t* d_err = nullptr;
  int32_t* d_hdr = nullptr;  // validation result of device-resident deltas
  int32_t* h_load = nullptr;  // pinned, kLoadRing slots of P values
  cudaEvent_t load_ev[kLoadRing] = {};
  // Copy streams of p2p_route_batch_host (inputs in, results out) and the events that order them.
  cudaStream_t cp_in = nullptr, cp_out = nullptr;
  // p2p_route_prepare: a batch whose grouping runs on grp_stream (low priority) while the next delta kernel
  // runs; the route of the same batch then waits for grp_done instead of grouping.
  struct Prepared {
    const int32_t* tokens = nullptr;
    const int64_t* offsets = nullptr;
    int64_t n_tokens = 0, B = 0;
    int state = 0;  // 0 none, 1 staged (grouping not launched yet), 2 launched on grp_stream
  } prep;
  cudaStream_t grp_stream = nullptr;
  cudaEvent_t grp_start = nullptr, grp_done = nullptr;
  cudaEvent_t ev_start = nullptr, ev_done = nullptr, ev_in[kPipe] = {}, ev_routed[kPipe] = {};
  int load_slot = 0;
  int32_t* h_err = nullptr;       // pinned
  TreeState* h_states = nullptr;  // pinned, P entries
  DevBuf req_tok, req_off, out_match, out_peer;
  DevBuf d_op, d_seg_begin, d_seg_off, d_seg_len, d_pool, d_peer_begin, d_done, d_gather;
  DevBuf grp_keys, grp_vals, grp_req, grp_ckpt;  // shared-prefix grouping of a batch
  DevBuf cmp_jobs, cmp_queue;          // device compaction
  DevBuf upd_cnt, upd_op, upd_sb, upd_so, upd_sl;  // a routed batch as an INSERT delta (p2p_update_estimates)
  DevBuf lru_buf;                                   // scratch of the LRU calls
  DevBuf gmemo;                                     // the delta kernel's launch-wide verified-run table
  DevBuf d_room;                                    // room bounds of the trees that stopped (room_kernel)
  DevBuf d_parts;                                   // the delta launch's CTA parts (split_trees)
  std::vector<int32_t> h_parts;                     // their host copy (kept until the next call)
  std::vector<uint8_t> lru;                         // per tree: kept as an LRU cache (p2p_lru_enable)
  std::vector<int64_t> lru_time;                    // per LRU tree: the time of its last insert or access
  int64_t launches = 0;  // kernels this router has launched
  RouterClock* clock = nullptr;  // per-kernel device time, while switched on
  // Shared label pool: long labels interned across trees (device array, host mirror, content index).
  int32_t* d_shared = nullptr;
  int64_t shared_cap = 0;
  std::vector<int32_t> h_shared;
  std::unordered_map<uint64_t, int32_t> intern;
  // Interned runs by a hash of their first kHeadTokens tokens: (pool offset, length), a few per head.
  std::unordered_map<uint64_t, std::vector<std::pair<int32_t, int32_t>>> heads;
  std::string err;
};

namespace {

// Makes the router's device current for the duration of a call, and installs its kernel clock (if on) on
// the calling thread.
struct DeviceGuard {
  int prev = -1;
  bool changed = false;
  p2p::KernelClock* prev_clock = nullptr;
  explicit DeviceGuard(const p2p_router* r) : DeviceGuard(r->device) {
    prev_clock = p2p::t_clock;
    p2p::t_clock = r->clock;
  }
  explicit DeviceGuard(int dev) {
    prev_clock = p2p::t_clock;
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) changed = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
    p2p::t_clock = prev_clock;
    if (changed) cudaSetDevice(prev);
  }
};

int fail(p2p_router* r, int code, const std::string& msg) {
  if (r)
    r->err = msg;
  else
    p2p::set_global_error(msg);
  return code;
}

int cuda_fail(p2p_router* r, cudaError_t e, const char* what) {
  return fail(r, P2P_E_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

#define CK(call)                                           \
  do {                                                     \
    cudaError_t e_ = (call);                               \
    if (e_ != cudaSuccess) return cuda_fail(r, e_, #call); \
  } while (0)

cudaError_t dalloc(p2p_router* r, void** p, size_t bytes) {
  return cudaMallocFromPoolAsync(p, bytes ? bytes : 16, r->pool, r->stream);
}
void dfree(p2p_router* r, void* p) {
  if (p) cudaFreeAsync(p, r->stream);
}

// Grow-only staging buffer.
cudaError_t ensure(p2p_router* r, DevBuf& b, size_t bytes) {
  if (b.cap >= bytes && b.p) return cudaSuccess;
  dfree(r, b.p);
  b.p = nullptr;
  b.cap = 0;
  const size_t cap = std::max(bytes + bytes / 4, (size_t)4096);
  cudaError_t e = dalloc(r, &b.p, cap);
  if (e == cudaSuccess) b.cap = cap;
  return e;
}

// Scratch of the shared-prefix grouping for a batch of B requests (B <= 2^30): a key table of at least 2B
// slots; slot_of, lead, cpre (B each), the two request lists (2B), gid, cmin and fcnt (B each) and eight counts;
// and checkpoint rows, as many as fit in 256 MB (and at most B/2 + 1, one per leader with followers).
cudaError_t group_scratch(p2p_router* r, int64_t B, p2p::GroupScratch& g) {
  const int64_t slots = std::max<int64_t>(next_pow2(2 * B), 1024);
  const int64_t gcap = std::max<int64_t>(1, std::min<int64_t>(B / 2 + 1, ((int64_t)256 << 20) / ((int64_t)r->P * 16)));
  cudaError_t e = ensure(r, r->grp_keys, (size_t)slots * sizeof(unsigned long long));
  if (e == cudaSuccess) e = ensure(r, r->grp_vals, (size_t)slots * sizeof(int32_t));
  if (e == cudaSuccess) e = ensure(r, r->grp_req, (size_t)(8 * B + 8) * sizeof(int32_t));
  if (e == cudaSuccess) e = ensure(r, r->grp_ckpt, (size_t)gcap * r->P * sizeof(int4));
  if (e != cudaSuccess) return e;
  int32_t* q = static_cast<int32_t*>(r->grp_req.p);
  g.keys = static_cast<unsigned long long*>(r->grp_keys.p);
  g.vals = static_cast<int32_t*>(r->grp_vals.p);
  g.bits = log2_exact(slots);
  g.slot_of = q;
  g.lead = q + B;
  g.cpre = q + 2 * B;
  g.lists = q + 3 * B;
  g.gid = q + 5 * B;
  g.cmin = q + 6 * B;
  g.fcnt = q + 7 * B;
  g.counts = q + 8 * B;
  g.ckpt = static_cast<int4*>(r->grp_ckpt.p);
  g.gcap = (int32_t)gcap;
  return cudaSuccess;
}

// Groups the batch by shared prefix and routes it (leaders, then followers).  The callers check B <= kMaxBatch
// (request indices and list positions are 32-bit).
// With decide (an excluded-peer mask staged with the load) or out_next, the passes make the decision with
// excluded trees and the next-best target.
int route(p2p_router* r, const int32_t* tokens, int64_t n_tokens, int64_t tok_base, const int64_t* offsets, int64_t B,
          int32_t alpha, int32_t* out_match, int32_t* out_peer, bool decide = false, int32_t* out_next = nullptr) {
  const auto& pr = r->prep;
  const bool same = pr.state != 0 && pr.tokens == tokens && pr.offsets == offsets && pr.n_tokens == n_tokens &&
                    pr.B == B && tok_base == 0;
  const bool grouped = same && pr.state == 2;
  if (r->prep.state == 2) CK(cudaStreamWaitEvent(r->stream, r->grp_done, 0));  // its scratch is this call's
  // (state 3, scratch taken but the grouping not launched, cannot outlive the delta call that took it)
  r->prep.state = 0;
  p2p::GroupScratch g;
  CK(group_scratch(r, B, g));
  if (!grouped) {
    CK(p2p::launch_group(tokens, n_tokens, tok_base, offsets, B, g, r->num_sms, r->stream));
    r->launches += 4;
  }
  int launched = 0;
  CK(p2p::launch_route(r->d_views, r->P, tokens, n_tokens, tok_base, offsets, B, r->d_load, alpha, out_match, out_peer,
                       r->d_err, &g, r->num_sms, r->stream, &launched, decide, out_next));
  r->launches += launched;
  return P2P_OK;
}

// A staged p2p_route_prepare grouping, in two steps around a delta kernel launch.  Before: its scratch is
// allocated (router-stream order) and grp_start marks the router stream there, ahead of the delta kernel.
// After: the grouping is launched on the side stream behind grp_start only, so it runs alongside the delta
// kernel, whose CTAs are resident first; the grouping uses the room they leave.
int prepare_scratch(p2p_router* r) {
  if (r->prep.state != 1) return P2P_OK;
  p2p::GroupScratch g;
  CK(group_scratch(r, r->prep.B, g));
  CK(cudaEventRecord(r->grp_start, r->stream));
  r->prep.state = 3;
  return P2P_OK;
}

int launch_prepared(p2p_router* r) {
  if (r->prep.state != 3) return P2P_OK;
  p2p::GroupScratch g;
  CK(group_scratch(r, r->prep.B, g));  // the buffers of prepare_scratch (no allocation)
  CK(cudaStreamWaitEvent(r->grp_stream, r->grp_start, 0));
  CK(p2p::launch_group(r->prep.tokens, r->prep.n_tokens, 0, r->prep.offsets, r->prep.B, g, r->num_sms, r->grp_stream));
  CK(cudaEventRecord(r->grp_done, r->grp_stream));
  r->launches += 4;
  r->prep.state = 2;
  return P2P_OK;
}

// Device-to-host copy ordered on the router stream (waits for it).
cudaError_t d2h(p2p_router* r, void* dst, const void* src, size_t bytes) {
  cudaError_t e = cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToHost, r->stream);
  return e == cudaSuccess ? cudaStreamSynchronize(r->stream) : e;
}

void free_tree_arrays(p2p_router* r, TreeState& t) {
  dfree(r, t.node);
  dfree(r, t.child);
  dfree(r, t.label);
  dfree(r, t.stamp);
  t.node = nullptr;
  t.child = nullptr;
  t.label = nullptr;
  t.stamp = nullptr;
}

// Allocates the arrays of a tree with the given capacities; on failure frees what it got.
cudaError_t alloc_tree_arrays(p2p_router* r, TreeState& t, int32_t cap_node, int32_t cap_child, int32_t cap_label) {
  t = TreeState{};
  cudaError_t e = dalloc(r, (void**)&t.node, (size_t)cap_node * sizeof(int4));
  if (e == cudaSuccess) e = dalloc(r, (void**)&t.child, (size_t)std::max(cap_child, 1) * sizeof(int4));
  if (e == cudaSuccess) e = dalloc(r, (void**)&t.label, (size_t)std::max(cap_label, 1) * sizeof(int32_t));
  if (e != cudaSuccess) {
    free_tree_arrays(r, t);
    return e;
  }
  t.cap_node = cap_node;
  t.cap_child = cap_child;
  t.cap_label = cap_label;
  return cudaSuccess;
}

int install_empty_tree(p2p_router* r, int32_t p) {
  TreeState t;
  const int32_t rb = table_bits_for(0, true);
  cudaError_t e = alloc_tree_arrays(r, t, 64, 4 << rb, 1024);
  if (e != cudaSuccess) return cuda_fail(r, e, "allocating an empty tree");
  const int4 root = make_int4(0, p2p::make_meta(rb, 0), 0, 0);
  CK(cudaMemsetAsync(t.child, 0, ((size_t)1 << rb) * sizeof(int4), r->stream));
  t.rfilter = r->d_rfilter + (size_t)p * p2p::kRootFilterWords;
  CK(cudaMemsetAsync(t.rfilter, 0, p2p::kRootFilterWords * sizeof(uint32_t), r->stream));
  CK(cudaMemcpyAsync(t.node, &root, sizeof(int4), cudaMemcpyHostToDevice, r->stream));
  CK(cudaStreamSynchronize(r->stream));  // `root` is a host temporary
  t.n_node = 1;
  t.n_child = 1 << rb;
  r->hs[(size_t)p] = t;
  CK(p2p::launch_set_tree(r->d_states + p, r->d_views + p, t, r->d_shared, r->stream));
  r->launches += 1;
  return P2P_OK;
}

int check_peer(p2p_router* r, int32_t peer) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (peer < 0 || peer >= r->P) return fail(r, P2P_E_INVAL, "peer " + std::to_string(peer) + " out of range");
  return P2P_OK;
}

int check_load(p2p_router* r, const int32_t* load, int32_t alpha) {
  if (!load) return fail(r, P2P_E_INVAL, "load is NULL");
  if (alpha < 0) return fail(r, P2P_E_INVAL, "alpha must be >= 0");
  for (int32_t p = 0; p < r->P; ++p) {
    if (load[p] < 0 || load[p] > 65535) return fail(r, P2P_E_INVAL, "load out of [0, 65535] for peer " + std::to_string(p));
    if ((int64_t)alpha * load[p] > INT32_MAX) return fail(r, P2P_E_INVAL, "alpha * load exceeds 2^31-1");
  }
  return P2P_OK;
}

// Stages load[P] through a pinned ring slot; with an excluded-peer mask (mask[p] != 0), tree p's load word
// also carries kLoadExcluded.  The slot's previous copy has finished once its event has.
int stage_load(p2p_router* r, const int32_t* load, const uint8_t* mask = nullptr) {
  const int s = r->load_slot;
  r->load_slot = (s + 1) % kLoadRing;
  CK(cudaEventSynchronize(r->load_ev[s]));
  int32_t* slot = r->h_load + (size_t)s * r->P;
  std::memcpy(slot, load, (size_t)r->P * sizeof(int32_t));
  if (mask)
    for (int32_t p = 0; p < r->P; ++p)
      if (mask[p]) slot[p] |= p2p::kLoadExcluded;
  CK(cudaMemcpyAsync(r->d_load, slot, (size_t)r->P * sizeof(int32_t), cudaMemcpyHostToDevice, r->stream));
  CK(cudaEventRecord(r->load_ev[s], r->stream));
  return P2P_OK;
}

int do_sync(p2p_router* r) {
  CK(cudaStreamSynchronize(r->stream));
  CK(cudaMemcpyAsync(r->h_err, r->d_err, sizeof(int32_t), cudaMemcpyDeviceToHost, r->stream));
  CK(cudaStreamSynchronize(r->stream));
  const int32_t bits = *r->h_err;
  if (bits) {
    CK(cudaMemsetAsync(r->d_err, 0, sizeof(int32_t), r->stream));
    CK(cudaStreamSynchronize(r->stream));
    std::string m = "device reported:";
    if (bits & p2p::ERR_BAD_OFFSETS) m += " request offsets outside [0, n_tokens] or decreasing;";
    if (bits & p2p::ERR_CORRUPT_TREE) m += " an inconsistent tree;";
    if (bits & p2p::ERR_STALL) m += " a route kernel wait timed out (outputs incomplete);";
    return fail(r, P2P_E_DEVICE, m);
  }
  return P2P_OK;
}

int push_states(p2p_router* r, int32_t p0, int32_t p1);

// Makes the device shared pool hold the host mirror's tokens [from, end): grows it (stream-ordered copy)
// if needed, in which case every tree's view is refreshed with the new pool address.
int sync_shared_pool(p2p_router* r, int64_t from) {
  const int64_t n = (int64_t)r->h_shared.size();
  if (n == from) return P2P_OK;
  if (n > r->shared_cap) {
    const int64_t cap = std::min<int64_t>(std::max<int64_t>(2 * r->shared_cap, n + (1 << 20)), INT32_MAX);
    int32_t* np = nullptr;
    cudaError_t e = dalloc(r, (void**)&np, (size_t)cap * sizeof(int32_t));
    if (e != cudaSuccess) return fail(r, P2P_E_NOMEM, std::string("growing the shared label pool: ") + cudaGetErrorString(e));
    if (from > 0) CK(cudaMemcpyAsync(np, r->d_shared, (size_t)from * sizeof(int32_t), cudaMemcpyDeviceToDevice, r->stream));
    dfree(r, r->d_shared);
    r->d_shared = np;
    r->shared_cap = cap;
    if (int rc = push_states(r, 0, r->P)) return rc;
    CK(p2p::launch_refresh_views(r->d_states, r->d_views, r->P, r->d_shared, r->stream));
    r->launches += 1;
  }
  CK(cudaMemcpyAsync(r->d_shared + from, r->h_shared.data() + from, (size_t)(n - from) * sizeof(int32_t),
                     cudaMemcpyHostToDevice, r->stream));
  CK(cudaStreamSynchronize(r->stream));  // the mirror may reallocate on the next append
  return P2P_OK;
}

// Interns a label of at least kInternMin tokens: an identical run, or a new run (whose head is then indexed).
// Returns its encoded offset, or 0 with ok = false (the pool is full).
int32_t intern_label(p2p_router* r, const int32_t* src, int32_t len, bool& ok) {
  ok = true;
  const uint64_t h = run_hash(src, len);
  auto it = r->intern.find(h);
  if (it != r->intern.end() && (int64_t)it->second + len <= (int64_t)r->h_shared.size() &&
      std::memcmp(r->h_shared.data() + it->second, src, (size_t)len * sizeof(int32_t)) == 0)
    return ~it->second;
  if ((int64_t)r->h_shared.size() + len >= INT32_MAX) {
    ok = false;
    return 0;
  }
  const int32_t at = (int32_t)r->h_shared.size();
  r->h_shared.insert(r->h_shared.end(), src, src + len);
  r->intern.emplace(h, at);
  auto& hs = r->heads[run_hash(src, kHeadTokens)];
  if (hs.size() < kHeadCandidates) hs.emplace_back(at, len);
  return ~at;
}

// The interned run sharing the longest prefix with src[0 .. len) among those indexed under the same head;
// k = that prefix's length (0: none).
int32_t longest_head(const p2p_router* r, const int32_t* src, int32_t len, int32_t& k) {
  k = 0;
  int32_t best = 0;
  auto it = r->heads.find(run_hash(src, kHeadTokens));
  if (it == r->heads.end()) return 0;
  for (const auto& [at, rl] : it->second) {
    const int32_t m = std::min(len, rl);
    const int32_t* a = r->h_shared.data() + at;
    const int32_t lcp = (int32_t)(std::mismatch(a, a + m, src).first - a);
    if (lcp > k) {
      k = lcp;
      best = at;
    }
  }
  return best;
}

int upload_flat(p2p_router* r, int32_t peer, const p2p_flat_tree* t) {
  std::string err;
  if (!p2p::validate_flat(t, err)) return fail(r, P2P_E_FORMAT, err);
  const int64_t N = t->n_nodes, NL = t->n_labels;
  // Labels: long runs are interned in the shared pool (label_off < 0 encodes pool offset ~off), the rest
  // go to the tree's own arena.  A long label whose first part (kInternMin tokens or more) starts an interned
  // run of another tree -- a prompt prefix that this tree holds with a single suffix, while other trees hold
  // it with several -- is split there: the edge takes the shared run's start, and a node with one child and
  // no sequence continues with the rest.  Every tree holding the prefix then points at one copy, so a walk
  // compares it once for all of them (and the export merges the node back).  A label that is a prefix of an
  // interned run points at that run.
  const int64_t shared_before = (int64_t)r->h_shared.size();
  std::vector<int32_t> enc((size_t)N, 0), head_len((size_t)N, 0), tail_enc((size_t)N, 0), own;
  own.reserve((size_t)NL);
  int64_t n_split = 0;
  for (int64_t v = 1; v < N; ++v) {
    const int32_t* src = t->labels + t->label_off[v];
    const int32_t len = t->label_len[v];
    bool interned = false;
    if (len >= kInternMin) {
      int32_t k = 0;
      const int32_t at = longest_head(r, src, len, k);
      if (k == len) {
        enc[(size_t)v] = ~at;
        interned = true;
      } else if (k >= kInternMin) {
        enc[(size_t)v] = ~at;
        head_len[(size_t)v] = k;
        ++n_split;
        const int32_t rest = len - k;
        bool ok = false;
        if (rest >= kInternMin) tail_enc[(size_t)v] = intern_label(r, src + k, rest, ok);
        if (!ok) {
          tail_enc[(size_t)v] = (int32_t)own.size();
          own.insert(own.end(), src + k, src + len);
        }
        interned = true;
      } else {
        enc[(size_t)v] = intern_label(r, src, len, interned);
      }
    }
    if (!interned) {
      enc[(size_t)v] = (int32_t)own.size();
      own.insert(own.end(), src, src + len);
    }
  }
  if (int rc = sync_shared_pool(r, shared_before)) return rc;
  // Children tables, laid out in node order in the child arena; the split nodes (ids N ..) after them.
  const int64_t NN = N + n_split;
  if (NN > INT32_MAX / 2) return fail(r, P2P_E_NOMEM, "too many nodes");
  std::vector<int32_t> bits((size_t)NN), off((size_t)NN, 0), split_id((size_t)N, 0);
  int64_t slots = 0;
  for (int64_t v = 0; v < N; ++v) {
    bits[(size_t)v] = table_bits_for(t->child_count[v], v == 0);
    if (bits[(size_t)v] > p2p::kMaxTabBits) return fail(r, P2P_E_NOMEM, "a node has too many children");
    off[(size_t)v] = (int32_t)slots;
    slots += bits[(size_t)v] ? (int64_t)1 << bits[(size_t)v] : 0;
    if (slots > INT32_MAX / 2) return fail(r, P2P_E_NOMEM, "children tables exceed the int32 arena");
  }
  for (int64_t v = 1, x = N; v < N; ++v)
    if (head_len[(size_t)v]) {
      split_id[(size_t)v] = (int32_t)x;
      bits[(size_t)x] = p2p::kMinTabBits;
      off[(size_t)x] = (int32_t)slots;
      slots += (int64_t)1 << p2p::kMinTabBits;
      if (slots > INT32_MAX / 2) return fail(r, P2P_E_NOMEM, "children tables exceed the int32 arena");
      ++x;
    }
  std::vector<int4> node((size_t)NN), child((size_t)slots, make_int4(0, 0, 0, 0));
  for (int64_t v = 0; v < N; ++v) {
    const int32_t cnt = t->child_count[v], b = bits[(size_t)v];
    node[(size_t)v] = make_int4(b ? off[(size_t)v] : 0, p2p::make_meta(b, cnt), cnt, t->term_count[v]);
    for (int64_t e = t->child_begin[v]; e < (int64_t)t->child_begin[v] + cnt; ++e) {
      const int32_t c = t->child_idx[e];
      const int32_t k = head_len[(size_t)c];
      if (!k) {
        table_put(child.data() + off[(size_t)v], b, make_int4(t->child_first_tok[e], c, enc[(size_t)c], t->label_len[c]));
        continue;
      }
      // v -> x (the shared head) -> c (the rest of the label).
      const int32_t x = split_id[(size_t)c];
      table_put(child.data() + off[(size_t)v], b, make_int4(t->child_first_tok[e], x, enc[(size_t)c], k));
      node[(size_t)x] = make_int4(off[(size_t)x], p2p::make_meta(p2p::kMinTabBits, 1), 1, 0);
      const int32_t* src = t->labels + t->label_off[c];
      table_put(child.data() + off[(size_t)x], p2p::kMinTabBits,
                make_int4(src[k], c, tail_enc[(size_t)c], t->label_len[c] - k));
    }
  }
  const int64_t n_own = (int64_t)own.size();
  // Headroom for device deltas (no regrowth for a few anti-entropy rounds of a few percent each).
  const int32_t cap_node = clamp_i32(2 * NN + 1024);
  const int32_t cap_child = clamp_i32(2 * slots + 1024);
  const int32_t cap_label = std::max(label_cap(n_own), clamp_i32(n_own + NL / 2));
  TreeState nt;
  cudaError_t e = alloc_tree_arrays(r, nt, cap_node, cap_child, cap_label);
  if (e != cudaSuccess) return fail(r, P2P_E_NOMEM, std::string("allocating the tree: ") + cudaGetErrorString(e));
  // The tree's spare set of arrays, a quarter larger than the live one (deltas grow the tree before it is
  // compacted): a later device compaction copies the tree into it, so the delta call that compacts maps no
  // new memory.  Without room for it there is none.
  TreeState& sp = r->spare[(size_t)peer];
  const int32_t sp_node = clamp_i32(cap_node + (int64_t)cap_node / 4),
                sp_child = clamp_i32(cap_child + (int64_t)cap_child / 4),
                sp_label = clamp_i32(cap_label + (int64_t)cap_label / 4);
  if (sp.cap_node < sp_node || sp.cap_child < sp_child || sp.cap_label < sp_label) {
    free_tree_arrays(r, sp);
    if (alloc_tree_arrays(r, sp, sp_node, sp_child, sp_label) != cudaSuccess) {
      sp = TreeState{};
      (void)cudaGetLastError();
    }
  }
  CK(cudaMemcpyAsync(nt.node, node.data(), (size_t)NN * sizeof(int4), cudaMemcpyHostToDevice, r->stream));
  if (slots) CK(cudaMemcpyAsync(nt.child, child.data(), (size_t)slots * sizeof(int4), cudaMemcpyHostToDevice, r->stream));
  if (n_own) CK(cudaMemcpyAsync(nt.label, own.data(), (size_t)n_own * sizeof(int32_t), cudaMemcpyHostToDevice, r->stream));
  nt.n_node = (int32_t)NN;
  nt.n_child = (int32_t)slots;
  nt.n_label = (int32_t)n_own;
  // The root's first-token filter: exactly the root's children now.
  std::vector<uint32_t> filt(p2p::kRootFilterWords, 0u);
  for (int64_t e = t->child_begin[0]; e < (int64_t)t->child_begin[0] + t->child_count[0]; ++e) {
    const uint32_t h = p2p::root_filter_bit(t->child_first_tok[e]);
    filt[h >> 5] |= 1u << (h & 31);
  }
  nt.rfilter = r->d_rfilter + (size_t)peer * p2p::kRootFilterWords;
  CK(cudaMemcpyAsync(nt.rfilter, filt.data(), filt.size() * sizeof(uint32_t), cudaMemcpyHostToDevice, r->stream));
  TreeState& old = r->hs[(size_t)peer];
  free_tree_arrays(r, old);
  old = nt;
  CK(p2p::launch_set_tree(r->d_states + peer, r->d_views + peer, nt, r->d_shared, r->stream));
  r->launches += 1;
  // The host vectors above are released on return; pageable copies have consumed them by now.
  return P2P_OK;
}

int download(p2p_router* r, int32_t peer, p2p_snapshot* out) {
  CK(cudaStreamSynchronize(r->stream));
  const TreeState& t = r->hs[(size_t)peer];
  std::vector<int4> node((size_t)t.n_node), child((size_t)t.n_child);
  std::vector<int32_t> label((size_t)t.n_label);
  if (t.n_node) CK(d2h(r, node.data(), t.node, node.size() * sizeof(int4)));
  if (t.n_child) CK(d2h(r, child.data(), t.child, child.size() * sizeof(int4)));
  if (t.n_label) CK(d2h(r, label.data(), t.label, label.size() * sizeof(int32_t)));
  std::string err;
  if (!p2p::snapshot_from_device_layout(node.data(), t.n_node, child.data(), t.n_child, label.data(), t.n_label,
                                        r->h_shared.data(), (int64_t)r->h_shared.size(), *out, err))
    return fail(r, P2P_E_DEVICE, err);
  return P2P_OK;
}

// Rebuilds tree p's root table (node 0's children) in fresh slots of the child arena, doubled (or, with
// extra > 0, sized for `extra` more children) and without tombstones.  Only the host does this: during a delta
// every warp of the tree shares the root table.
int regrow_root(p2p_router* r, int32_t p, int64_t extra = 0) {
  TreeState& t = r->hs[(size_t)p];
  int4 root;
  CK(d2h(r, &root, t.node, sizeof(int4)));
  const int32_t bits = p2p::tab_bits(root.y);
  std::vector<int4> tab(bits ? (size_t)1 << bits : 0);
  if (bits) CK(d2h(r, tab.data(), t.child + root.x, tab.size() * sizeof(int4)));
  std::vector<int4> kids;
  for (const int4& s : tab)
    if (s.y >= 1) kids.push_back(s);
  const int32_t nb = std::max(bits + 1, table_bits_for((int64_t)kids.size() + extra, true));
  if (nb > p2p::kMaxTabBits) return fail(r, P2P_E_NOMEM, "root table too large");
  const int64_t n_slots = (int64_t)1 << nb;
  if ((int64_t)t.cap_child - t.n_child < n_slots) {
    t.need_child = (int32_t)n_slots;
    t.need_root = 0;
    return 1;  // the caller grows the child arena first, then comes back
  }
  std::vector<int4> nt((size_t)n_slots, make_int4(0, 0, 0, 0));
  for (const int4& k : kids) table_put(nt.data(), nb, k);
  const int4 nr = make_int4(t.n_child, p2p::make_meta(nb, (int32_t)kids.size()), (int32_t)kids.size(), root.w);
  CK(cudaMemcpyAsync(t.child + t.n_child, nt.data(), (size_t)n_slots * sizeof(int4), cudaMemcpyHostToDevice, r->stream));
  CK(cudaMemcpyAsync(t.node, &nr, sizeof(int4), cudaMemcpyHostToDevice, r->stream));
  CK(cudaStreamSynchronize(r->stream));  // nt and nr are host temporaries
  t.stale_child += bits ? (int64_t)1 << bits : 0;
  t.n_child += (int32_t)n_slots;
  return P2P_OK;
}

// Grows the arenas of tree p so that the largest op that did not fit does (at least doubling them), or, with
// whole, so that need_* -- the room the rest of the call may take -- fits with an eighth to spare.
int grow_tree(p2p_router* r, int32_t p, bool whole = false) {
  TreeState& t = r->hs[(size_t)p];
  auto newcap = [whole](int64_t cap, int64_t used, int64_t need) -> int64_t {
    if (whole) return std::max<int64_t>(cap, used + need + std::max<int64_t>(need / 8, 1024));
    return std::max<int64_t>(cap * 2, used + 2 * need + 1024);
  };
  bool grow_n = (int64_t)t.cap_node - t.n_node < t.need_node;
  bool grow_c = (int64_t)t.cap_child - t.n_child < t.need_child;
  bool grow_l = (int64_t)t.cap_label - t.n_label < t.need_label;
  if (!grow_n && !grow_c && !grow_l && !t.need_root) grow_n = grow_c = grow_l = true;  // always make progress
  if ((grow_n && (int64_t)t.n_node + t.need_node > INT32_MAX) ||
      (grow_c && (int64_t)t.n_child + t.need_child > INT32_MAX) ||
      (grow_l && (int64_t)t.n_label + t.need_label > INT32_MAX))
    return fail(r, P2P_E_NOMEM, "tree " + std::to_string(p) + " outgrows the int32 arena indices");
  const int64_t cn = grow_n ? std::min<int64_t>(newcap(t.cap_node, t.n_node, t.need_node), INT32_MAX) : t.cap_node;
  const int64_t cc = grow_c ? std::min<int64_t>(newcap(t.cap_child, t.n_child, t.need_child), INT32_MAX) : t.cap_child;
  const int64_t cl = grow_l ? std::min<int64_t>(newcap(t.cap_label, t.n_label, t.need_label), INT32_MAX) : t.cap_label;
  int4* nn = t.node;
  int4* nc = t.child;
  int32_t* nl = t.label;
  cudaError_t e = cudaSuccess;
  if (grow_n && e == cudaSuccess) e = dalloc(r, (void**)&nn, (size_t)cn * sizeof(int4));
  if (grow_c && e == cudaSuccess) e = dalloc(r, (void**)&nc, (size_t)cc * sizeof(int4));
  if (grow_l && e == cudaSuccess) e = dalloc(r, (void**)&nl, (size_t)cl * sizeof(int32_t));
  if (e != cudaSuccess) {
    if (nn != t.node) dfree(r, nn);
    if (nc != t.child) dfree(r, nc);
    if (nl != t.label) dfree(r, nl);
    return fail(r, P2P_E_NOMEM, std::string("growing a tree: ") + cudaGetErrorString(e));
  }
  if (grow_n) {
    CK(cudaMemcpyAsync(nn, t.node, (size_t)t.n_node * sizeof(int4), cudaMemcpyDeviceToDevice, r->stream));
    dfree(r, t.node);
    if (t.stamp) {  // an LRU tree's stamps follow its node slots; new slots start at time 0
      uint32_t* ns = nullptr;
      CK(dalloc(r, (void**)&ns, (size_t)cn * sizeof(uint32_t)));
      CK(cudaMemcpyAsync(ns, t.stamp, (size_t)t.n_node * sizeof(uint32_t), cudaMemcpyDeviceToDevice, r->stream));
      CK(cudaMemsetAsync(ns + t.n_node, 0, (size_t)(cn - t.n_node) * sizeof(uint32_t), r->stream));
      dfree(r, t.stamp);
      t.stamp = ns;
    }
  }
  if (grow_c) {
    CK(cudaMemcpyAsync(nc, t.child, (size_t)t.n_child * sizeof(int4), cudaMemcpyDeviceToDevice, r->stream));
    dfree(r, t.child);
  }
  if (grow_l) {
    CK(cudaMemcpyAsync(nl, t.label, (size_t)t.n_label * sizeof(int32_t), cudaMemcpyDeviceToDevice, r->stream));
    dfree(r, t.label);
  }
  t.node = nn;
  t.child = nc;
  t.label = nl;
  t.cap_node = (int32_t)cn;
  t.cap_child = (int32_t)cc;
  t.cap_label = (int32_t)cl;
  if (t.need_root) {
    int rc = regrow_root(r, p);
    if (rc == 1) {  // the child arena had no room for the new root table: grow it, then retry
      t.need_node = t.need_label = 0;
      t.need_root = 1;
      rc = grow_tree(r, p);
    }
    if (rc != P2P_OK) return rc;
  }
  t.status = p2p::DELTA_OK;
  t.need_node = t.need_child = t.need_label = t.need_root = 0;
  return P2P_OK;
}

// Before a delta of many INSERTs: a tree whose root table would pass 1/2 claimed with `ins[p - p0]` more
// children gets a root table sized for them now (growing its child arena first if needed), so the delta kernel
// does not stop and relaunch once per doubling.  Reads the roots of those trees (one copy each, one wait).
int presize_roots(p2p_router* r, int32_t p0, int32_t p1, const int64_t* ins) {
  std::vector<int32_t> ps;
  for (int32_t p = p0; p < p1; ++p)
    if (ins[p - p0] >= 1024) ps.push_back(p);
  if (ps.empty()) return P2P_OK;
  std::vector<int4> roots(ps.size());
  for (size_t i = 0; i < ps.size(); ++i)
    CK(cudaMemcpyAsync(&roots[i], r->hs[(size_t)ps[i]].node, sizeof(int4), cudaMemcpyDeviceToHost, r->stream));
  CK(cudaStreamSynchronize(r->stream));
  for (size_t i = 0; i < ps.size(); ++i) {
    const int32_t p = ps[i];
    const int64_t extra = ins[p - p0];
    if (!p2p::tab_full(p2p::tab_bits(roots[i].y), (int64_t)p2p::tab_used(roots[i].y) + extra)) continue;
    int rc = regrow_root(r, p, extra);
    if (rc == 1) {  // the child arena has no room for the new table: grow it first
      TreeState& t = r->hs[(size_t)p];
      t.need_node = t.need_label = 0;
      t.need_root = 0;
      rc = grow_tree(r, p);
      if (rc == P2P_OK) rc = regrow_root(r, p, extra);
    }
    if (rc != P2P_OK) return rc == 1 ? fail(r, P2P_E_NOMEM, "no room for a root table") : rc;
  }
  return push_states(r, p0, p1);
}

// Rebuilds a tree whose arenas are mostly stale entries: canonical export, then a fresh upload.
int compact_tree(p2p_router* r, int32_t p) {
  p2p_snapshot snap;
  int rc = download(r, p, &snap);
  if (rc != P2P_OK) return rc;
  p2p_flat_tree v;
  p2p_snapshot_view(&snap, &v);
  return upload_flat(r, p, &v);
}

// Compacts trees ps on the device: fresh arrays sized from the live counts with the same headroom as an
// upload; compact_kernel copies each tree's structure (one CTA per tree) and compact_labels_kernel moves all
// their labels over the whole GPU; then the states and views of [p0, p1) are republished.  A tree
// whose fresh arrays turn out too small keeps its old arrays and is compacted through the host instead.
int compact_trees(p2p_router* r, const std::vector<int32_t>& ps, int32_t p0, int32_t p1) {
  if (ps.empty()) return P2P_OK;
  const size_t n = ps.size();
  std::vector<p2p::CompactJob> jobs(n);
  std::vector<TreeState> fresh(n);
  std::vector<char> from_spare(n, 0);
  // Fresh arrays that are not used after all: a spare goes back to its tree, the rest to the pool.
  auto release = [&](size_t j) {
    if (from_spare[j])
      r->spare[(size_t)ps[j]] = fresh[j];
    else
      free_tree_arrays(r, fresh[j]);
  };
  std::vector<int64_t> qoff(n);
  int64_t qtotal = 0;
  int32_t max_cap_node = 0;
  for (size_t i = 0; i < n; ++i) {
    const TreeState& t = r->hs[(size_t)ps[i]];
    const int64_t nodes = std::max<int64_t>((int64_t)t.n_node - t.dead_nodes, 1);
    const int64_t slots = std::max<int64_t>((int64_t)t.n_child - t.stale_child, 0);
    const int64_t own = std::max<int64_t>((int64_t)t.n_label - t.stale_label, 0);
    const int32_t cn = clamp_i32(2 * nodes + 1024), cc = clamp_i32(2 * slots + 1024), cl = label_cap(own);
    // The spare serves when it holds the live tree with a quarter to spare; growth ahead of later calls
    // (apply_delta) adds room from there.
    TreeState& sp = r->spare[(size_t)ps[i]];
    if (sp.node && sp.cap_node >= nodes + nodes / 4 + 1024 && sp.cap_child >= slots + slots / 4 + 1024 &&
        sp.cap_label >= own + own / 4 + 65536) {
      fresh[i] = sp;
      from_spare[i] = 1;
      sp = TreeState{};
    } else {
      cudaError_t e = alloc_tree_arrays(r, fresh[i], cn, cc, cl);
      if (e != cudaSuccess) {
        for (size_t j = 0; j < i; ++j) release(j);
        return fail(r, P2P_E_NOMEM, std::string("allocating a compacted tree: ") + cudaGetErrorString(e));
      }
    }
    const TreeState& f = fresh[i];
    jobs[i] = p2p::CompactJob{t.node, t.child, t.label, f.node, f.child, f.label, nullptr,
                              f.cap_node, f.cap_child, f.cap_label, 0, 0, 0, 0, 0};
    qoff[i] = qtotal;
    qtotal += f.cap_node;
    max_cap_node = std::max(max_cap_node, f.cap_node);
  }
  CK(ensure(r, r->cmp_queue, (size_t)qtotal * sizeof(int4)));
  CK(ensure(r, r->cmp_jobs, n * sizeof(p2p::CompactJob)));
  for (size_t i = 0; i < n; ++i) jobs[i].queue = static_cast<int4*>(r->cmp_queue.p) + qoff[i];
  CK(cudaMemcpyAsync(r->cmp_jobs.p, jobs.data(), n * sizeof(p2p::CompactJob), cudaMemcpyHostToDevice, r->stream));
  CK(p2p::launch_compact(static_cast<p2p::CompactJob*>(r->cmp_jobs.p), (int32_t)n, max_cap_node, r->num_sms,
                         r->stream));
  r->launches += 2;
  CK(d2h(r, jobs.data(), r->cmp_jobs.p, n * sizeof(p2p::CompactJob)));
  std::vector<int32_t> retry;
  for (size_t i = 0; i < n; ++i) {
    TreeState& t = r->hs[(size_t)ps[i]];
    if (jobs[i].status != 0) {
      release(i);
      retry.push_back(ps[i]);
      continue;
    }
    // The old arrays become the tree's spare (a smaller spare goes back to the pool).
    TreeState& sp = r->spare[(size_t)ps[i]];
    free_tree_arrays(r, sp);
    sp = TreeState{};
    sp.node = t.node;
    sp.child = t.child;
    sp.label = t.label;
    sp.cap_node = t.cap_node;
    sp.cap_child = t.cap_child;
    sp.cap_label = t.cap_label;
    t = fresh[i];
    t.n_node = jobs[i].n_node;
    t.n_child = jobs[i].n_child;
    t.n_label = jobs[i].n_label;
  }
  if (int rc = push_states(r, p0, p1)) return rc;
  CK(p2p::launch_refresh_views(r->d_states + p0, r->d_views + p0, p1 - p0, r->d_shared, r->stream));
  r->launches += 1;
  for (int32_t p : retry)
    if (int rc = compact_tree(r, p)) return rc;
  return P2P_OK;
}

bool needs_compaction(const TreeState& t) {
  if (t.stamp) return false;  // LRU trees are not compacted (their stamps are indexed by node slot)
  return (t.stale_label > 65536 && 2 * t.stale_label > t.n_label) ||
         (t.stale_child > 65536 && 2 * t.stale_child > t.n_child) ||
         (t.dead_nodes > 16384 && 2 * t.dead_nodes > t.n_node);
}

// A tree at least 70% of the way to needs_compaction.  When some tree of a call is compacted, these go
// along in the same launch: replicas that receive deltas at the same rate reach the threshold within a few
// calls of one another, and one compaction wave costs about as much as one of a handful of trees.
bool nears_compaction(const TreeState& t) {
  if (t.stamp) return false;
  return (t.stale_label > 45875 && 20 * t.stale_label > 7 * (int64_t)t.n_label) ||
         (t.stale_child > 45875 && 20 * t.stale_child > 7 * (int64_t)t.n_child) ||
         (t.dead_nodes > 11468 && 20 * t.dead_nodes > 7 * (int64_t)t.n_node);
}

// Resets the per-call fields of trees [p0, p1) and copies their states to the device.
int push_states(p2p_router* r, int32_t p0, int32_t p1) {
  for (int32_t p = p0; p < p1; ++p) r->hs[(size_t)p].rfilter = r->d_rfilter + (size_t)p * p2p::kRootFilterWords;
  std::memcpy(r->h_states, r->hs.data() + p0, (size_t)(p1 - p0) * sizeof(TreeState));
  CK(cudaMemcpyAsync(r->d_states + p0, r->h_states, (size_t)(p1 - p0) * sizeof(TreeState), cudaMemcpyHostToDevice,
                     r->stream));
  CK(cudaStreamSynchronize(r->stream));  // h_states is reused right after
  return P2P_OK;
}

int pull_states(p2p_router* r, int32_t p0, int32_t p1) {
  CK(cudaMemcpyAsync(r->h_states, r->d_states + p0, (size_t)(p1 - p0) * sizeof(TreeState), cudaMemcpyDeviceToHost,
                     r->stream));
  CK(cudaStreamSynchronize(r->stream));
  std::memcpy(r->hs.data() + p0, r->h_states, (size_t)(p1 - p0) * sizeof(TreeState));
  return P2P_OK;
}

// A delta may not give ops to an LRU tree (its stamps change only through the p2p_lru_* calls).  With
// peer = -1, the ranges of the LRU trees are read from peer_begin (host, or two words copied back each).
int reject_lru_ops(p2p_router* r, int32_t peer, const p2p_delta* d) {
  const int32_t p0 = peer == -1 ? 0 : peer, p1 = peer == -1 ? r->P : peer + 1;
  for (int32_t p = p0; p < p1; ++p) {
    if (!r->lru[(size_t)p]) continue;
    int64_t n = d->seqs.n;
    if (peer == -1) {
      int64_t pb[2] = {0, 0};
      if (d->mem == P2P_MEM_HOST) {
        pb[0] = d->peer_begin[p];
        pb[1] = d->peer_begin[p + 1];
      } else {
        CK(cudaMemcpyAsync(pb, d->peer_begin + p, sizeof(pb), cudaMemcpyDeviceToHost, r->stream));
        CK(cudaStreamSynchronize(r->stream));
      }
      n = pb[1] - pb[0];
    }
    if (n != 0)
      return fail(r, P2P_E_INVAL, "tree " + std::to_string(p) + " is an LRU tree: it changes only through the p2p_lru_* calls");
  }
  return P2P_OK;
}

}  // namespace

extern "C" {

int p2p_router_create(int32_t P, p2p_router** out) {
  if (!out) return fail(nullptr, P2P_E_INVAL, "out is NULL");
  *out = nullptr;
  if (P < 1 || P > 65536) return fail(nullptr, P2P_E_INVAL, "P must be in [1, 65536]");
  p2p_router* r = new p2p_router();
  r->P = P;
  auto bail = [&](int code) {
    p2p::set_global_error(r->err);
    p2p_router_destroy(r);
    return code;
  };
  cudaError_t e = cudaGetDevice(&r->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&r->num_sms, cudaDevAttrMultiProcessorCount, r->device);
  if (e != cudaSuccess) {
    cuda_fail(r, e, "querying the device");
    return bail(P2P_E_CUDA);
  }
  cudaMemPoolProps props = {};
  props.allocType = cudaMemAllocationTypePinned;
  props.location.type = cudaMemLocationTypeDevice;
  props.location.id = r->device;
  e = cudaMemPoolCreate(&r->pool, &props);
  if (e == cudaSuccess) {
    uint64_t keep = UINT64_MAX;  // keep freed blocks in the pool: re-uploads reuse them
    e = cudaMemPoolSetAttribute(r->pool, cudaMemPoolAttrReleaseThreshold, &keep);
  }
  if (e != cudaSuccess) {
    cuda_fail(r, e, "creating the memory pool");
    return bail(P2P_E_CUDA);
  }
  r->hs.assign((size_t)P, TreeState{});
  r->spare.assign((size_t)P, TreeState{});
  r->lru.assign((size_t)P, 0);
  r->lru_time.assign((size_t)P, 0);
  e = dalloc(r, (void**)&r->d_views, (size_t)P * sizeof(TreeView));
  if (e == cudaSuccess) e = dalloc(r, (void**)&r->d_states, (size_t)P * sizeof(TreeState));
  if (e == cudaSuccess) e = dalloc(r, (void**)&r->d_rfilter, (size_t)P * p2p::kRootFilterWords * sizeof(uint32_t));
  if (e == cudaSuccess) e = dalloc(r, (void**)&r->d_load, (size_t)P * sizeof(int32_t));
  if (e == cudaSuccess) e = dalloc(r, (void**)&r->d_err, sizeof(int32_t));
  if (e == cudaSuccess) e = dalloc(r, (void**)&r->d_hdr, p2p::kStaticHeaderInts * sizeof(int32_t));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&r->h_load, (size_t)kLoadRing * P * sizeof(int32_t));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&r->h_err, sizeof(int32_t));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&r->h_states, (size_t)P * sizeof(TreeState));
  for (int i = 0; i < kLoadRing && e == cudaSuccess; ++i) e = cudaEventCreateWithFlags(&r->load_ev[i], cudaEventDisableTiming);
  if (e == cudaSuccess) {
    int lo = 0, hi = 0;  // the side stream of prepared groupings yields to the router's kernels
    e = cudaDeviceGetStreamPriorityRange(&lo, &hi);
    if (e == cudaSuccess) e = cudaStreamCreateWithPriority(&r->grp_stream, cudaStreamNonBlocking, lo);
  }
  for (cudaEvent_t* ev : {&r->grp_start, &r->grp_done})
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(ev, cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&r->cp_in, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&r->cp_out, cudaStreamNonBlocking);
  for (cudaEvent_t* ev : {&r->ev_start, &r->ev_done})
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(ev, cudaEventDisableTiming);
  for (int i = 0; i < kPipe && e == cudaSuccess; ++i) {
    e = cudaEventCreateWithFlags(&r->ev_in[i], cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&r->ev_routed[i], cudaEventDisableTiming);
  }
  if (e == cudaSuccess) e = cudaMemsetAsync(r->d_err, 0, sizeof(int32_t), r->stream);
  if (e != cudaSuccess) {
    fail(r, P2P_E_NOMEM, std::string("allocating router state: ") + cudaGetErrorString(e));
    return bail(P2P_E_NOMEM);
  }
  for (int32_t p = 0; p < P; ++p) {
    const int rc = install_empty_tree(r, p);
    if (rc != P2P_OK) return bail(rc);
  }
  e = cudaStreamSynchronize(r->stream);
  if (e != cudaSuccess) {
    cuda_fail(r, e, "initialising trees");
    return bail(P2P_E_CUDA);
  }
  *out = r;
  return P2P_OK;
}

void p2p_router_destroy(p2p_router* r) {
  if (!r) return;
  DeviceGuard g(r);
  cudaStreamSynchronize(r->stream);
  for (cudaStream_t s : {r->cp_in, r->cp_out, r->grp_stream})  // copies or a prepared grouping in flight
    if (s) cudaStreamSynchronize(s);
  if (r->pool) {
    for (TreeState& t : r->hs) free_tree_arrays(r, t);
    for (TreeState& t : r->spare) free_tree_arrays(r, t);
    for (DevBuf* b : {&r->req_tok, &r->req_off, &r->out_match, &r->out_peer, &r->d_op, &r->d_seg_begin,
                      &r->d_seg_off, &r->d_seg_len, &r->d_pool, &r->d_peer_begin, &r->d_done, &r->d_gather,
                      &r->grp_keys, &r->grp_vals, &r->grp_req, &r->grp_ckpt, &r->cmp_jobs, &r->cmp_queue,
                      &r->upd_cnt, &r->upd_op, &r->upd_sb, &r->upd_so, &r->upd_sl, &r->lru_buf, &r->gmemo,
                      &r->d_room, &r->d_parts})
      dfree(r, b->p);
    dfree(r, r->d_views);
    dfree(r, r->d_states);
    dfree(r, r->d_rfilter);
    dfree(r, r->d_load);
    dfree(r, r->d_err);
    dfree(r, r->d_hdr);
    dfree(r, r->d_shared);
    cudaStreamSynchronize(r->stream);
    cudaMemPoolDestroy(r->pool);
  }
  for (cudaEvent_t ev : r->load_ev)
    if (ev) cudaEventDestroy(ev);
  for (cudaStream_t s : {r->cp_in, r->cp_out, r->grp_stream})
    if (s) {
      cudaStreamSynchronize(s);
      cudaStreamDestroy(s);
    }
  for (cudaEvent_t ev : {r->grp_start, r->grp_done})
    if (ev) cudaEventDestroy(ev);
  for (cudaEvent_t ev : {r->ev_start, r->ev_done})
    if (ev) cudaEventDestroy(ev);
  for (int i = 0; i < kPipe; ++i) {
    if (r->ev_in[i]) cudaEventDestroy(r->ev_in[i]);
    if (r->ev_routed[i]) cudaEventDestroy(r->ev_routed[i]);
  }
  if (r->h_load) cudaFreeHost(r->h_load);
  if (r->h_err) cudaFreeHost(r->h_err);
  if (r->h_states) cudaFreeHost(r->h_states);
  delete r->clock;
  delete r;
}

int p2p_router_set_stream(p2p_router* r, void* stream) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  DeviceGuard g(r);
  CK(cudaStreamSynchronize(r->stream));
  r->stream = (cudaStream_t)stream;
  return P2P_OK;
}

int p2p_router_sync(p2p_router* r) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  DeviceGuard g(r);
  return do_sync(r);
}

const char* p2p_last_error(const p2p_router* r) { return r ? r->err.c_str() : p2p::global_error(); }

int32_t p2p_router_num_trees(const p2p_router* r) { return r ? r->P : 0; }

int64_t p2p_router_launch_count(const p2p_router* r) { return r ? r->launches : 0; }

int p2p_router_kernel_clock(p2p_router* r, int32_t on) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  DeviceGuard g(r->device);
  CK(cudaStreamSynchronize(r->stream));
  if (on) {
    if (!r->clock) r->clock = new RouterClock();
    r->clock->reset();
  } else if (r->clock) {
    r->clock->resolve();
    delete r->clock;
    r->clock = nullptr;
  }
  return P2P_OK;
}

int p2p_router_kernel_time(p2p_router* r, int32_t i, const char** name, int64_t* launches, double* ms) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (i < 0 || i >= p2p::K_COUNT_) return fail(r, P2P_E_INVAL, "kernel index out of range");
  if (name) *name = p2p::kernel_name(i);
  int64_t n = 0;
  double t = 0.0;
  if (r->clock) {
    DeviceGuard g(r->device);
    CK(cudaStreamSynchronize(r->stream));
    r->clock->resolve();
    if (r->clock->err != cudaSuccess) return cuda_fail(r, r->clock->err, "kernel clock");
    n = r->clock->n[i];
    t = r->clock->ms[i];
  }
  if (launches) *launches = n;
  if (ms) *ms = t;
  return P2P_OK;
}

int p2p_tree_upload(p2p_router* r, int32_t peer, const p2p_flat_tree* t) {
  if (int rc = check_peer(r, peer)) return rc;
  if (r->lru[(size_t)peer]) return fail(r, P2P_E_INVAL, "an LRU tree changes only through the p2p_lru_* calls");
  DeviceGuard g(r);
  return upload_flat(r, peer, t);
}

int p2p_tree_build(p2p_router* r, int32_t peer, const p2p_seqs* seqs) {
  if (int rc = check_peer(r, peer)) return rc;
  if (r->lru[(size_t)peer]) return fail(r, P2P_E_INVAL, "an LRU tree changes only through the p2p_lru_* calls");
  std::string err;
  if (!seqs || !p2p::check_seqs(seqs, err, nullptr, nullptr)) return fail(r, P2P_E_INVAL, seqs ? err : "seqs is NULL");
  p2p_snapshot snap;
  if (!p2p::build_snapshot(*seqs, snap, err)) return fail(r, P2P_E_NOMEM, err);
  p2p_flat_tree v;
  p2p_snapshot_view(&snap, &v);
  DeviceGuard g(r);
  return upload_flat(r, peer, &v);
}

int p2p_tree_download(p2p_router* r, int32_t peer, p2p_snapshot** out) {
  if (int rc = check_peer(r, peer)) return rc;
  if (!out) return fail(r, P2P_E_INVAL, "out is NULL");
  *out = nullptr;
  DeviceGuard g(r);
  p2p_snapshot* s = new p2p_snapshot();
  const int rc = download(r, peer, s);
  if (rc != P2P_OK) {
    p2p_snapshot_free(s);
    return rc;
  }
  *out = s;
  return P2P_OK;
}

int p2p_tree_stats(p2p_router* r, int32_t peer, int64_t out[9]) {
  if (int rc = check_peer(r, peer)) return rc;
  if (!out) return fail(r, P2P_E_INVAL, "out is NULL");
  DeviceGuard g(r);
  CK(cudaStreamSynchronize(r->stream));
  const TreeState& t = r->hs[(size_t)peer];
  const int64_t v[9] = {(int64_t)t.n_node - t.dead_nodes, t.n_node, t.n_child, t.n_label, t.stale_child,
                        t.stale_label, t.cap_node, t.cap_child, t.cap_label};
  std::memcpy(out, v, sizeof(v));
  return P2P_OK;
}

static int apply_delta_impl(p2p_router* r, int32_t peer, const p2p_delta* d, int64_t* n_absent, bool lru_ok);

int p2p_tree_apply_delta(p2p_router* r, int32_t peer, const p2p_delta* d, int64_t* n_absent) {
  return apply_delta_impl(r, peer, d, n_absent, false);
}

// The CTAs of a delta launch.  A CTA takes the ops of one tree, except that a tree with many more ops than a
// CTA's share of the call -- the call's ops over the SMs, and at least kPartOps -- is split into up to
// kDeltaBuckets parts by first-token bucket, so that it does not hold the whole launch on one SM (a batch
// routed mostly to one tree and inserted with p2p_update_estimates, for one).  n_blocks = nt and
// d_parts = NULL when no tree is split.
constexpr int64_t kPartOps = 16384;
static int split_trees(p2p_router* r, int32_t peer, const p2p_delta* d, const int64_t* d_pb, int32_t p0, int32_t nt,
                int64_t n, int32_t& n_blocks, const int32_t*& d_parts) {
  n_blocks = nt;
  d_parts = nullptr;
  const int64_t share = std::max<int64_t>((n + r->num_sms - 1) / std::max(r->num_sms, 1), kPartOps);
  if (n <= share) return P2P_OK;
  std::vector<int64_t> ops((size_t)nt, n);
  if (peer == -1) {
    std::vector<int64_t> pb((size_t)r->P + 1);
    if (d->mem == P2P_MEM_HOST) {
      std::memcpy(pb.data(), d->peer_begin, pb.size() * sizeof(int64_t));
    } else {
      CK(d2h(r, pb.data(), d_pb, pb.size() * sizeof(int64_t)));
    }
    for (int32_t i = 0; i < nt; ++i) ops[(size_t)i] = pb[(size_t)i + 1] - pb[(size_t)i];
  }
  std::vector<int32_t>& w = r->h_parts;
  w.clear();
  for (int32_t i = 0; i < nt; ++i) {
    const int32_t np = (int32_t)std::min<int64_t>(p2p::kDeltaBuckets, (ops[(size_t)i] + share - 1) / share);
    for (int32_t c = 0; c < std::max(np, 1); ++c)
      w.push_back(i | c << p2p::kPartShift | std::max(np, 1) << p2p::kNpartShift);
  }
  if ((int32_t)w.size() == nt) return P2P_OK;
  CK(ensure(r, r->d_parts, w.size() * sizeof(int32_t)));
  CK(cudaMemcpyAsync(r->d_parts.p, w.data(), w.size() * sizeof(int32_t), cudaMemcpyHostToDevice, r->stream));
  n_blocks = (int32_t)w.size();
  d_parts = static_cast<const int32_t*>(r->d_parts.p);
  return P2P_OK;
}

static int apply_delta_impl(p2p_router* r, int32_t peer, const p2p_delta* d, int64_t* n_absent, bool lru_ok) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (peer < -1 || peer >= r->P) return fail(r, P2P_E_INVAL, "peer out of range");
  if (!d) return fail(r, P2P_E_INVAL, "delta is NULL");
  if (d->mem != P2P_MEM_HOST && d->mem != P2P_MEM_DEVICE) return fail(r, P2P_E_INVAL, "delta.mem must be HOST or DEVICE");
  DeviceGuard g(r);
  const p2p_seqs& S = d->seqs;
  const int64_t n = S.n;
  if (n < 0 || S.n_segs < 0 || S.n_pool < 0) return fail(r, P2P_E_INVAL, "negative size in delta");
  if (n > 0 && (!d->op || !S.seg_begin || (S.n_segs > 0 && (!S.seg_off || !S.seg_len)) || (S.n_pool > 0 && !S.pool)))
    return fail(r, P2P_E_INVAL, "NULL array in delta");
  if (peer == -1 && n > 0 && !d->peer_begin) return fail(r, P2P_E_INVAL, "peer = -1 needs peer_begin");
  if (n == 0) {
    if (n_absent) *n_absent = 0;
    return P2P_OK;
  }
  const int32_t p0 = peer == -1 ? 0 : peer, p1 = peer == -1 ? r->P : peer + 1;
  const int32_t nt = p1 - p0;
  if (!lru_ok)
    if (int rc = reject_lru_ops(r, peer, d)) return rc;
  int64_t max_len = 0, max_runs = 0;
  const int32_t* d_op = d->op;
  const int64_t *d_sb = S.seg_begin, *d_so = S.seg_off, *d_pb = d->peer_begin;
  const int32_t *d_sl = S.seg_len, *d_pool = S.pool;
  p2p_delta dv = *d;  // the delta as the device reads it
  if (d->mem == P2P_MEM_HOST) {
    // Host arrays are copied as they are into device buffers and validated there like a device-resident
    // delta: one pass over millions of ops on the GPU instead of a scan on the host.
    CK(ensure(r, r->d_op, (size_t)n * sizeof(int32_t)));
    CK(ensure(r, r->d_seg_begin, (size_t)(n + 1) * sizeof(int64_t)));
    CK(ensure(r, r->d_seg_off, (size_t)std::max<int64_t>(S.n_segs, 1) * sizeof(int64_t)));
    CK(ensure(r, r->d_seg_len, (size_t)std::max<int64_t>(S.n_segs, 1) * sizeof(int32_t)));
    CK(ensure(r, r->d_pool, (size_t)std::max<int64_t>(S.n_pool, 1) * sizeof(int32_t)));
    CK(cudaMemcpyAsync(r->d_op.p, d->op, (size_t)n * sizeof(int32_t), cudaMemcpyHostToDevice, r->stream));
    CK(cudaMemcpyAsync(r->d_seg_begin.p, S.seg_begin, (size_t)(n + 1) * sizeof(int64_t), cudaMemcpyHostToDevice, r->stream));
    if (S.n_segs) {
      CK(cudaMemcpyAsync(r->d_seg_off.p, S.seg_off, (size_t)S.n_segs * sizeof(int64_t), cudaMemcpyHostToDevice, r->stream));
      CK(cudaMemcpyAsync(r->d_seg_len.p, S.seg_len, (size_t)S.n_segs * sizeof(int32_t), cudaMemcpyHostToDevice, r->stream));
    }
    if (S.n_pool) CK(cudaMemcpyAsync(r->d_pool.p, S.pool, (size_t)S.n_pool * sizeof(int32_t), cudaMemcpyHostToDevice, r->stream));
    if (peer == -1) {
      CK(ensure(r, r->d_peer_begin, (size_t)(r->P + 1) * sizeof(int64_t)));
      CK(cudaMemcpyAsync(r->d_peer_begin.p, d->peer_begin, (size_t)(r->P + 1) * sizeof(int64_t), cudaMemcpyHostToDevice,
                         r->stream));
      dv.peer_begin = (const int64_t*)r->d_peer_begin.p;
    }
    dv.op = (const int32_t*)r->d_op.p;
    dv.seqs.seg_begin = (const int64_t*)r->d_seg_begin.p;
    dv.seqs.seg_off = (const int64_t*)r->d_seg_off.p;
    dv.seqs.seg_len = (const int32_t*)r->d_seg_len.p;
    dv.seqs.pool = (const int32_t*)r->d_pool.p;
    dv.mem = P2P_MEM_DEVICE;
    d_op = dv.op;
    d_sb = dv.seqs.seg_begin;
    d_so = dv.seqs.seg_off;
    d_sl = dv.seqs.seg_len;
    d_pool = dv.seqs.pool;
    d_pb = dv.peer_begin;
  }
  {
    // Validate on the device; only the 16-byte result comes back.
    CK(p2p::launch_validate(r->d_hdr, &dv, peer, r->P, r->stream));
    r->launches += 1;
    int32_t h[4] = {0, 0, 0, 0};
    CK(d2h(r, h, r->d_hdr, sizeof(h)));
    unsigned long long ml = 0;
    std::memcpy(&ml, h, sizeof(ml));
    max_len = (int64_t)ml;
    max_runs = h[3];
    if (h[2] & p2p::STATIC_BAD_OP) return fail(r, P2P_E_INVAL, "bad op code in the delta");
    if (h[2] & p2p::STATIC_BAD_SEGMENT) return fail(r, P2P_E_INVAL, "seg_begin or a segment is malformed or outside the pool");
    if (h[2] & p2p::STATIC_TOO_LONG) return fail(r, P2P_E_INVAL, "a sequence is longer than 2^31-1 tokens");
    if (h[2] & p2p::STATIC_BAD_PEER_BEGIN) return fail(r, P2P_E_INVAL, "peer_begin must run non-decreasing from 0 to n");
  }
  CK(ensure(r, r->d_done, (size_t)std::max<int64_t>(n, 1)));
  // A tree with many more ops than a CTA's share of the call is split among CTAs (delta_kernel's parts).
  int32_t n_blocks = nt;
  const int32_t* d_parts = nullptr;
  if (int e = split_trees(r, peer, d, d_pb, p0, nt, n, n_blocks, d_parts)) return e;
  int32_t* gather = nullptr;
  const int64_t stride = std::max<int64_t>(max_len, 1);
  if (max_runs > 2) {
    CK(ensure(r, r->d_gather, (size_t)n_blocks * p2p::kDeltaWarps * stride * sizeof(int32_t)));
    gather = (int32_t*)r->d_gather.p;
  }
  uint8_t* done = (uint8_t*)r->d_done.p;
  std::vector<int4> before((size_t)nt);  // arena use at the start of the call
  for (int32_t p = p0; p < p1; ++p) {
    const TreeState& t = r->hs[(size_t)p];
    before[(size_t)(p - p0)] = make_int4(t.n_node, t.n_child, t.n_label, 0);
  }
  // Device states = host mirror, then this call's op ranges (set on the device) and cleared done flags.
  if (int rc = push_states(r, p0, p1)) return rc;
  CK(p2p::launch_init_ranges(r->d_states + p0, nt, peer == -1 ? d_pb : nullptr, n, r->stream));
  if (n) CK(cudaMemsetAsync(done, 0, (size_t)n, r->stream));
  r->launches += 1;
  // The launch-wide verified-run table, cleared for this call (labels and the pool do not change during it).
  const size_t gslots = (size_t)1 << p2p::kGlobalMemoBits;
  CK(ensure(r, r->gmemo, gslots * (sizeof(unsigned long long) + sizeof(int32_t))));
  p2p::GlobalMemo gm{static_cast<unsigned long long*>(r->gmemo.p),
                     reinterpret_cast<int32_t*>(static_cast<unsigned long long*>(r->gmemo.p) + gslots),
                     (uint32_t)(gslots - 1)};
  CK(cudaMemsetAsync(r->gmemo.p, 0, gslots * (sizeof(unsigned long long) + sizeof(int32_t)), r->stream));
  int rc = P2P_OK;
  bool sized = false;  // the room of the rest of the call was bounded once (room_kernel)
  for (int round = 0;; ++round) {
    if (round == 64) {
      rc = fail(r, P2P_E_NOMEM, "delta did not fit after 64 arena growths");
      break;
    }
    if (round == 0)
      if (int rc = prepare_scratch(r)) return rc;
    CK(p2p::launch_delta(r->d_states + p0, done, nt, d_op, d_sb, d_so, d_sl, d_pool, gather, stride, r->d_shared,
                         r->stream, &gm, d_parts, n_blocks));
    if (round == 0)
      if (int rc = launch_prepared(r)) return rc;  // a prepared batch's grouping overlaps the delta kernel
    r->launches += 1;
    if (int e = pull_states(r, p0, p1)) return e;
    bool again = false, stopped = false;
    for (int32_t p = p0; p < p1; ++p) stopped = stopped || (r->hs[(size_t)p].status & p2p::DELTA_NEED_SPACE);
    // The first stop for room: the room every op not yet applied may take, per tree (room_kernel), so that a
    // tree is grown once for the rest of the call (a delta that brings many new sequences to one tree would
    // otherwise stop at every doubling).  The bound counts INSERTs only; a later stop (a DELETE's fold needs
    // label room too) grows by the largest op that did not fit, as before.
    std::vector<long long> room;
    if (stopped && !sized) {
      sized = true;
      CK(ensure(r, r->d_room, (size_t)nt * 2 * sizeof(long long)));
      CK(p2p::launch_room(r->d_states + p0, nt, done, d_op, d_sb, d_sl, static_cast<long long*>(r->d_room.p),
                          r->stream));
      r->launches += 1;
      room.resize((size_t)nt * 2);
      CK(d2h(r, room.data(), r->d_room.p, room.size() * sizeof(long long)));
    }
    for (int32_t p = p0; p < p1 && rc == P2P_OK; ++p) {
      TreeState& t = r->hs[(size_t)p];
      if (t.status & p2p::DELTA_CORRUPT) {
        rc = fail(r, P2P_E_DEVICE, "tree " + std::to_string(p) + " is inconsistent");
      } else if (t.status & p2p::DELTA_NEED_SPACE) {
        bool whole = false;
        if (!room.empty()) {
          const long long tok = room[(size_t)(p - p0) * 2], ins = room[(size_t)(p - p0) * 2 + 1];
          const auto bound = [](long long want, int32_t used) {
            return (int32_t)std::min<long long>(want, (long long)INT32_MAX / 2 - used);
          };
          if (t.need_label) t.need_label = std::max(t.need_label, bound(tok, t.n_label));
          if (t.need_node) t.need_node = std::max(t.need_node, bound(2 * ins + 64, t.n_node));
          if (t.need_child) t.need_child = std::max(t.need_child, bound(8 * ins + 1024, t.n_child));
          whole = true;
        }
        rc = grow_tree(r, p, whole);
        again = true;
      }
    }
    if (rc != P2P_OK || !again) break;
    if (int e = push_states(r, p0, p1)) return e;
  }
  // Room ahead of the next call: free room in an arena below twice what this call used there.  Such a tree is
  // grown now, so the next call's kernel does not stop for room -- unless it is compacted in this call.
  // A wave of compaction starts when a tree is past the threshold, or when a tree near it is short of room
  // (compaction hands it arrays with headroom, where growth would copy its stale space only to be replaced by
  // a compaction a call or two later); every tree near the threshold goes along.
  std::vector<int4> short_of((size_t)nt, make_int4(0, 0, 0, 0));  // (node, child, label room wanted, any)
  bool wave = false;
  for (int32_t p = p0; p < p1; ++p) {
    const TreeState& t = r->hs[(size_t)p];
    const int4 b = before[(size_t)(p - p0)];
    const int64_t dn = 2 * std::max<int64_t>((int64_t)t.n_node - b.x, 0);
    const int64_t dc = 2 * std::max<int64_t>((int64_t)t.n_child - b.y, 0);
    const int64_t dl = 2 * std::max<int64_t>((int64_t)t.n_label - b.z, 0);
    const bool short_n = (int64_t)t.cap_node - t.n_node < dn, short_c = (int64_t)t.cap_child - t.n_child < dc,
               short_l = (int64_t)t.cap_label - t.n_label < dl;
    const bool is_short = short_n || short_c || short_l;
    short_of[(size_t)(p - p0)] = make_int4(short_n ? clamp_i32(dn) : 0, short_c ? clamp_i32(dc) : 0,
                                           short_l ? clamp_i32(dl) : 0, is_short);
    wave = wave || needs_compaction(t) || (is_short && nears_compaction(t));
  }
  std::vector<int32_t> stale;
  for (int32_t p = p0; wave && p < p1; ++p)
    if (nears_compaction(r->hs[(size_t)p])) stale.push_back(p);  // (a tree past the threshold is near it)
  for (int32_t p = p0, k = 0; p < p1 && rc == P2P_OK; ++p) {
    if (k < (int32_t)stale.size() && stale[(size_t)k] == p) {
      ++k;
      continue;
    }
    const int4 s = short_of[(size_t)(p - p0)];
    if (!s.w) continue;
    TreeState& t = r->hs[(size_t)p];
    t.need_node = s.x;
    t.need_child = s.y;
    t.need_label = s.z;
    t.need_root = 0;
    rc = grow_tree(r, p);
  }
  // Publish the (possibly moved) arrays to the route kernel's view table; compact the stale trees.
  if (int e = push_states(r, p0, p1)) return e;
  CK(p2p::launch_refresh_views(r->d_states + p0, r->d_views + p0, nt, r->d_shared, r->stream));
  r->launches += 1;
  int64_t absent = 0;
  for (int32_t p = p0; p < p1; ++p) absent += r->hs[(size_t)p].n_absent;
  if (rc == P2P_OK) rc = compact_trees(r, stale, p0, p1);
  if (n_absent) *n_absent = absent;
  return rc;
}

// The delta call for callers that cannot allocate (see the header and delta_static.cu): device-resident
// delta, validation on the device, scratch in the library's static device array, no arena growth and no
// compaction.
int p2p_tree_apply_delta_static(p2p_router* r, int32_t peer, const p2p_delta* d, int64_t* n_absent) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (peer < -1 || peer >= r->P) return fail(r, P2P_E_INVAL, "peer out of range");
  if (!d) return fail(r, P2P_E_INVAL, "delta is NULL");
  if (d->mem != P2P_MEM_DEVICE) return fail(r, P2P_E_INVAL, "p2p_tree_apply_delta_static needs a delta in device memory");
  const p2p_seqs& S = d->seqs;
  if (S.n < 0 || S.n_segs < 0 || S.n_pool < 0) return fail(r, P2P_E_INVAL, "negative size in delta");
  if (S.n > 0 && (!d->op || !S.seg_begin || (S.n_segs > 0 && (!S.seg_off || !S.seg_len)) || (S.n_pool > 0 && !S.pool)))
    return fail(r, P2P_E_INVAL, "NULL array in delta");
  if (peer == -1 && S.n > 0 && !d->peer_begin) return fail(r, P2P_E_INVAL, "peer = -1 needs peer_begin");
  DeviceGuard g(r);
  if (S.n > 0)
    if (int rc = reject_lru_ops(r, peer, d)) return rc;
  int32_t* header = nullptr;
  int32_t* tokens = nullptr;
  CK(p2p::static_scratch(r->device, &header, &tokens));
  if (S.n == 0) {
    if (n_absent) *n_absent = 0;
    return P2P_OK;
  }
  CK(p2p::launch_validate(header, d, peer, r->P, r->stream));
  r->launches += 1;
  int32_t h[4] = {0, 0, 0, 0};
  CK(cudaMemcpyAsync(h, header, sizeof(h), cudaMemcpyDeviceToHost, r->stream));
  CK(cudaStreamSynchronize(r->stream));
  unsigned long long max_len = 0;
  std::memcpy(&max_len, h, sizeof(max_len));
  const int32_t bits = h[2], max_runs = h[3];
  if (bits & p2p::STATIC_BAD_OP) return fail(r, P2P_E_INVAL, "bad op code in the delta");
  if (bits & p2p::STATIC_BAD_SEGMENT) return fail(r, P2P_E_INVAL, "seg_begin or a segment is malformed or outside the pool");
  if (bits & p2p::STATIC_TOO_LONG) return fail(r, P2P_E_INVAL, "a sequence is longer than 2^31-1 tokens");
  if (bits & p2p::STATIC_BAD_PEER_BEGIN) return fail(r, P2P_E_INVAL, "peer_begin must run non-decreasing from 0 to n");
  const int32_t p0 = peer == -1 ? 0 : peer, p1 = peer == -1 ? r->P : peer + 1;
  const int32_t nt = p1 - p0;
  // Scratch: one done byte per op (in whole words); gathered sequences only when an op has > 2 pool runs.
  const int64_t done_ints = (S.n + 3) / 4;
  const int64_t stride = max_len > 0 ? (int64_t)max_len : 1;
  const int64_t gather_ints = max_runs > 2 ? (int64_t)nt * p2p::kDeltaWarps * stride : 0;
  if (done_ints + gather_ints > p2p::static_scratch_tokens())
    return fail(r, P2P_E_INVAL, "the delta needs " + std::to_string(done_ints + gather_ints) +
                                    " words of scratch, more than the static scratch of " +
                                    std::to_string(p2p::static_scratch_tokens()) +
                                    " (exceeds the static scratch: split the delta or its sequences' runs)");
  uint8_t* done = reinterpret_cast<uint8_t*>(tokens);
  int32_t* gather = gather_ints ? tokens + done_ints : nullptr;
  CK(p2p::launch_init_ranges(r->d_states + p0, nt, peer == -1 ? d->peer_begin : nullptr, S.n, r->stream));
  if (S.n) CK(cudaMemsetAsync(done, 0, (size_t)S.n, r->stream));
  CK(p2p::launch_delta(r->d_states + p0, done, nt, d->op, S.seg_begin, S.seg_off, S.seg_len, S.pool, gather, stride,
                       r->d_shared, r->stream));
  r->launches += 2;
  CK(cudaMemcpyAsync(r->h_states, r->d_states + p0, (size_t)nt * sizeof(TreeState), cudaMemcpyDeviceToHost, r->stream));
  CK(cudaStreamSynchronize(r->stream));
  std::memcpy(r->hs.data() + p0, r->h_states, (size_t)nt * sizeof(TreeState));
  int rc = P2P_OK;
  int64_t absent = 0;
  for (int32_t p = p0; p < p1; ++p) {
    const TreeState& t = r->hs[(size_t)p];
    absent += t.n_absent;
    if (rc != P2P_OK) continue;
    if (t.status & p2p::DELTA_CORRUPT)
      rc = fail(r, P2P_E_DEVICE, "tree " + std::to_string(p) + " is inconsistent");
    else if (t.status & p2p::DELTA_NEED_SPACE)
      rc = fail(r, P2P_E_NOMEM, "tree " + std::to_string(p) +
                                    " ran out of arena room: some of its ops were not applied (p2p_tree_apply_delta grows trees)");
  }
  if (n_absent) *n_absent = absent;
  return rc;
}

// UpdateTrieEstimate / UpdateTrie of Algorithm 1 over a routed batch: the batch is counting-sorted by its
// chosen tree into an INSERT delta in router buffers (update_kernel.cu), whose ops are runs of the request
// tokens, and applied by the delta path.
int p2p_update_estimates(p2p_router* r, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets, int64_t B,
                         const int32_t* peer, int64_t* n_inserted) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (n_inserted) *n_inserted = 0;
  if (B < 0 || n_tokens < 0) return fail(r, P2P_E_INVAL, "negative B or n_tokens");
  if (B > kMaxBatch) return fail(r, P2P_E_INVAL, "B exceeds 2^30 requests per call: split the batch");
  if (B == 0) return P2P_OK;
  if (!offsets || !peer || (n_tokens > 0 && !tokens)) return fail(r, P2P_E_INVAL, "NULL device pointer");
  DeviceGuard g(r);
  const int32_t P = r->P;
  // counts [P] int32 | cursor [P] int32 | bad [2] int32 | peer_begin [P+1] int64 | total [1] int64
  const size_t cnt_bytes = ((size_t)2 * P + 2) * sizeof(int32_t);
  CK(ensure(r, r->upd_cnt, cnt_bytes + (size_t)(P + 2) * sizeof(int64_t)));
  int32_t* counts = static_cast<int32_t*>(r->upd_cnt.p);
  int32_t* cursor = counts + P;
  int32_t* bad = cursor + P;
  int64_t* peer_begin = reinterpret_cast<int64_t*>(static_cast<char*>(r->upd_cnt.p) + cnt_bytes);
  int64_t* total = peer_begin + P + 1;
  CK(ensure(r, r->upd_sb, (size_t)(B + 1) * sizeof(int64_t)));
  int64_t* seg_begin = static_cast<int64_t*>(r->upd_sb.p);
  CK(cudaMemsetAsync(counts, 0, cnt_bytes, r->stream));
  CK(p2p::launch_update_count(peer, offsets, B, n_tokens, P, counts, bad, r->num_sms, r->stream));
  CK(p2p::launch_update_scan(counts, P, peer_begin, cursor, seg_begin + B, total, r->stream));
  r->launches += 2;
  struct {
    int32_t bad[2];
    int64_t total;
  } h = {};
  std::vector<int64_t> pb((size_t)P + 1);
  CK(cudaMemcpyAsync(h.bad, bad, sizeof(h.bad), cudaMemcpyDeviceToHost, r->stream));
  CK(cudaMemcpyAsync(&h.total, total, sizeof(h.total), cudaMemcpyDeviceToHost, r->stream));
  CK(cudaMemcpyAsync(pb.data(), peer_begin, pb.size() * sizeof(int64_t), cudaMemcpyDeviceToHost, r->stream));
  CK(cudaStreamSynchronize(r->stream));
  if (h.bad[0] & 1) return fail(r, P2P_E_INVAL, "a peer index is >= P");
  if (h.bad[0] & 2) return fail(r, P2P_E_INVAL, "a routed request has offsets outside [0, n_tokens] or decreasing");
  const int64_t n = h.total;
  if (n == 0) return P2P_OK;
  // Every op is an INSERT: a tree that takes many (the fresh prompts of a batch all go to its least-loaded
  // tree) gets its root table sized for them before the delta kernel runs.
  std::vector<int64_t> ins((size_t)P);
  for (int32_t p = 0; p < P; ++p) {
    ins[(size_t)p] = pb[(size_t)p + 1] - pb[(size_t)p];
    if (ins[(size_t)p] && r->lru[(size_t)p])
      return fail(r, P2P_E_INVAL, "requests routed to LRU tree " + std::to_string(p) + " go in through p2p_lru_insert");
  }
  if (int rc = presize_roots(r, 0, P, ins.data())) return rc;
  CK(ensure(r, r->upd_op, (size_t)n * sizeof(int32_t)));
  CK(ensure(r, r->upd_so, (size_t)n * sizeof(int64_t)));
  CK(ensure(r, r->upd_sl, (size_t)n * sizeof(int32_t)));
  int32_t* op = static_cast<int32_t*>(r->upd_op.p);
  int64_t* seg_off = static_cast<int64_t*>(r->upd_so.p);
  int32_t* seg_len = static_cast<int32_t*>(r->upd_sl.p);
  // seg_begin[n] = n was written by the scan at seg_begin + B: move it to its place when n < B.
  if (n < B) CK(cudaMemcpyAsync(seg_begin + n, seg_begin + B, sizeof(int64_t), cudaMemcpyDeviceToDevice, r->stream));
  CK(p2p::launch_update_scatter(peer, offsets, B, n_tokens, P, cursor, op, seg_begin, seg_off, seg_len, r->num_sms,
                                r->stream));
  r->launches += 1;
  p2p_delta d = {};
  d.op = op;
  d.seqs.n = n;
  d.seqs.seg_begin = seg_begin;
  d.seqs.seg_off = seg_off;
  d.seqs.seg_len = seg_len;
  d.seqs.pool = tokens;
  d.seqs.n_segs = n;
  d.seqs.n_pool = n_tokens;
  d.peer_begin = peer_begin;
  d.mem = P2P_MEM_DEVICE;
  const int rc = p2p_tree_apply_delta(r, -1, &d, nullptr);
  if (rc == P2P_OK && n_inserted) *n_inserted = n;
  return rc;
}

// ---- LRU trees: EvictLRUTrie of Algorithm 1 with device stamps (lru_kernel.cu) ----------------------------

static int check_lru(p2p_router* r, int32_t tree, int64_t time) {
  if (int rc = check_peer(r, tree)) return rc;
  if (!r->lru[(size_t)tree]) return fail(r, P2P_E_INVAL, "tree " + std::to_string(tree) + " is not an LRU tree");
  if (time < r->lru_time[(size_t)tree] || time > (int64_t)0xFFFFFFFE)
    return fail(r, P2P_E_INVAL, "time must not decrease and must be at most 2^32 - 2");
  return P2P_OK;
}

// An access at `time`: PrefixMatch of every request, the touched nodes stamped, partially touched edges split.
static int lru_access_impl(p2p_router* r, int32_t tree, const int32_t* tokens, int64_t n_tokens,
                           const int64_t* offsets, int64_t B, int64_t time, int32_t* out_match) {
  TreeState& t = r->hs[(size_t)tree];
  // Room for one split (a node and a 4-slot table) per request.
  const bool short_n = (int64_t)t.cap_node - t.n_node < B, short_c = (int64_t)t.cap_child - t.n_child < 4 * B;
  if (short_n || short_c) {
    if ((int64_t)t.n_node + B > INT32_MAX || (int64_t)t.n_child + 4 * B > INT32_MAX)
      return fail(r, P2P_E_NOMEM, "the LRU tree would outgrow the int32 arena indices");
    t.need_node = short_n ? clamp_i32(B) : 0;
    t.need_child = short_c ? clamp_i32(4 * B) : 0;
    t.need_label = 0;
    t.need_root = 0;
    if (int rc = grow_tree(r, tree)) return rc;
  }
  const int32_t n0 = t.n_node;
  CK(ensure(r, r->lru_buf, (size_t)2 * n0 * sizeof(int32_t)));
  int32_t* touch = static_cast<int32_t*>(r->lru_buf.p);
  int32_t* pslot = touch + n0;
  CK(cudaMemsetAsync(touch, 0, (size_t)n0 * sizeof(int32_t), r->stream));
  if (int rc = push_states(r, tree, tree + 1)) return rc;
  CK(p2p::launch_lru_walk(t, r->d_shared, tokens, n_tokens, offsets, B, touch, pslot, out_match, r->d_err, r->num_sms,
                          r->stream));
  CK(p2p::launch_lru_stamp(t, r->d_states + tree, r->d_shared, touch, pslot, n0, (uint32_t)time, r->num_sms,
                           r->stream));
  if (int rc = pull_states(r, tree, tree + 1)) return rc;
  CK(p2p::launch_refresh_views(r->d_states + tree, r->d_views + tree, 1, r->d_shared, r->stream));
  r->launches += 3;
  r->lru_time[(size_t)tree] = time;
  return P2P_OK;
}

int p2p_lru_enable(p2p_router* r, int32_t tree) {
  if (int rc = check_peer(r, tree)) return rc;
  if (r->lru[(size_t)tree]) return P2P_OK;
  DeviceGuard g(r);
  TreeState& t = r->hs[(size_t)tree];
  CK(cudaStreamSynchronize(r->stream));
  uint32_t* st = nullptr;
  cudaError_t e = dalloc(r, (void**)&st, (size_t)std::max(t.cap_node, 1) * sizeof(uint32_t));
  if (e != cudaSuccess) return fail(r, P2P_E_NOMEM, std::string("allocating stamps: ") + cudaGetErrorString(e));
  CK(cudaMemsetAsync(st, 0, (size_t)std::max(t.cap_node, 1) * sizeof(uint32_t), r->stream));
  t.stamp = st;
  r->lru[(size_t)tree] = 1;
  r->lru_time[(size_t)tree] = 0;
  return push_states(r, tree, tree + 1);
}

int p2p_lru_access(p2p_router* r, int32_t tree, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets,
                   int64_t B, int64_t time, int32_t* out_match) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (int rc = check_lru(r, tree, time)) return rc;
  if (B < 0 || n_tokens < 0 || B > kMaxBatch) return fail(r, P2P_E_INVAL, "B or n_tokens out of range");
  if (B == 0) return P2P_OK;
  if (!offsets || (n_tokens > 0 && !tokens)) return fail(r, P2P_E_INVAL, "NULL device pointer");
  DeviceGuard g(r);
  return lru_access_impl(r, tree, tokens, n_tokens, offsets, B, time, out_match);
}

int p2p_lru_insert(p2p_router* r, int32_t tree, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets,
                   int64_t B, int64_t time) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (int rc = check_lru(r, tree, time)) return rc;
  if (B < 0 || n_tokens < 0 || B > kMaxBatch) return fail(r, P2P_E_INVAL, "B or n_tokens out of range");
  if (B == 0) return P2P_OK;
  if (!offsets || (n_tokens > 0 && !tokens)) return fail(r, P2P_E_INVAL, "NULL device pointer");
  DeviceGuard g(r);
  CK(ensure(r, r->upd_op, (size_t)B * sizeof(int32_t)));
  CK(ensure(r, r->upd_sb, (size_t)(B + 1) * sizeof(int64_t)));
  CK(ensure(r, r->upd_so, (size_t)B * sizeof(int64_t)));
  CK(ensure(r, r->upd_sl, (size_t)B * sizeof(int32_t)));
  int32_t* op = static_cast<int32_t*>(r->upd_op.p);
  int64_t* sb = static_cast<int64_t*>(r->upd_sb.p);
  int64_t* so = static_cast<int64_t*>(r->upd_so.p);
  int32_t* sl = static_cast<int32_t*>(r->upd_sl.p);
  CK(p2p::launch_lru_ops(offsets, B, n_tokens, op, sb, so, sl, r->num_sms, r->stream));
  r->launches += 1;
  p2p_delta d = {};
  d.op = op;
  d.seqs.n = B;
  d.seqs.seg_begin = sb;
  d.seqs.seg_off = so;
  d.seqs.seg_len = sl;
  d.seqs.pool = tokens;
  d.seqs.n_segs = B;
  d.seqs.n_pool = n_tokens;
  d.mem = P2P_MEM_DEVICE;
  // UpdateTrie: the sequences go in (invalid offsets fail validation: nothing changes), then every token of
  // their paths is touched at `time`.
  if (int rc = apply_delta_impl(r, tree, &d, nullptr, true)) return rc;
  return lru_access_impl(r, tree, tokens, n_tokens, offsets, B, time, nullptr);
}

int p2p_lru_evict(p2p_router* r, int32_t tree, int64_t n_tokens, int64_t* n_evicted) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (n_evicted) *n_evicted = 0;
  if (int rc = check_peer(r, tree)) return rc;
  if (!r->lru[(size_t)tree]) return fail(r, P2P_E_INVAL, "tree " + std::to_string(tree) + " is not an LRU tree");
  if (n_tokens < 0) return fail(r, P2P_E_INVAL, "negative n_tokens");
  if (n_tokens == 0) return P2P_OK;
  DeviceGuard g(r);
  const TreeState& t = r->hs[(size_t)tree];
  const int64_t N = std::max<int32_t>(t.n_node, 1);
  // Scratch, per node slot: order, parent, cslot, end, surv (int32); size, off, rank, best (64-bit); gone; two
  // counters; then the sibling-offset sort (a power of two of entries at least N - 1: key, scan 64-bit; val;
  // and first per node slot).
  int64_t n2 = 1;
  while (n2 < N - 1) n2 <<= 1;
  const size_t main_bytes = ((size_t)N * (5 * 4 + 4 * 8 + 1) + 64 + 15) & ~(size_t)15;
  const size_t bytes = main_bytes + (size_t)n2 * (8 + 8 + 4) + (size_t)N * 4;
  CK(ensure(r, r->lru_buf, bytes));
  char* base = static_cast<char*>(r->lru_buf.p);
  p2p::LruSortScratch sc;
  sc.key = reinterpret_cast<unsigned long long*>(base + main_bytes);
  sc.scan = reinterpret_cast<int64_t*>(sc.key + n2);
  sc.val = reinterpret_cast<int32_t*>(sc.scan + n2);
  sc.first = sc.val + n2;
  int64_t* size = reinterpret_cast<int64_t*>(base);
  int64_t* off = size + N;
  int64_t* rank = off + N;
  unsigned long long* best = reinterpret_cast<unsigned long long*>(rank + N);
  unsigned long long* ctr = best + N;                      // [0]: token count, [1]: the BFS frontier size
  int32_t* order = reinterpret_cast<int32_t*>(ctr + 2);
  int32_t* parent = order + N;
  int32_t* cslot = parent + N;
  int32_t* end = cslot + N;
  int32_t* surv = end + N;
  uint8_t* gone = reinterpret_cast<uint8_t*>(surv + N);
  int32_t* n_next = reinterpret_cast<int32_t*>(ctr + 1);
  // Breadth-first order of the live nodes, level by level (order[0] = the root).
  CK(cudaMemsetAsync(order, 0, sizeof(int32_t), r->stream));
  std::vector<int32_t> lvl{0, 1};
  for (;;) {
    const int32_t l = (int32_t)lvl.size() - 2;
    CK(cudaMemsetAsync(n_next, 0, sizeof(int32_t), r->stream));
    CK(p2p::launch_lru_bfs(t, order + lvl[(size_t)l], lvl[(size_t)l + 1] - lvl[(size_t)l], order + lvl[(size_t)l + 1],
                           n_next, (int32_t)(N - lvl[(size_t)l + 1]), parent, cslot, r->num_sms, r->stream));
    r->launches += 1;
    int32_t h = 0;
    CK(d2h(r, &h, n_next, sizeof(h)));
    if (h == 0) break;
    if ((int64_t)lvl.back() + h > N) return fail(r, P2P_E_DEVICE, "the LRU tree is inconsistent");
    lvl.push_back(lvl.back() + h);
  }
  const int32_t n_levels = (int32_t)lvl.size() - 1, total = lvl.back();
  CK(p2p::launch_lru_init(order, total, size, off, rank, best, gone, r->num_sms, r->stream));
  CK(p2p::launch_lru_levels(t, order, lvl.data(), n_levels, parent, cslot, size, off, rank, best, end, sc, r->num_sms,
                            r->stream));
  {
    int64_t stages = 0, m = total - 1, k2 = 1;
    for (int32_t lg = 0; k2 < m; ++lg, k2 <<= 1) stages += lg + 1;  // bitonic steps: L (L + 1) / 2 for n2 = 2^L
    r->launches += 1 + 3 * (n_levels - 1) + (m > 0 ? 4 + stages : 0);
  }
  auto count = [&](int mode, uint32_t S, unsigned long long K, unsigned long long& out) -> int {
    CK(p2p::launch_lru_count(t, order + 1, total - 1, cslot, rank, end, mode, S, K, ctr, r->num_sms, r->stream));
    r->launches += 1;
    CK(d2h(r, &out, ctr, sizeof(out)));
    return P2P_OK;
  };
  // The threshold: stamps first, then the (end rank, deeper first) key inside the boundary stamp.
  unsigned long long all = 0, c = 0;
  if (int rc = count(0, 0xFFFFFFFFu, 0, all)) return rc;
  uint32_t S = 0xFFFFFFFFu;
  unsigned long long K = 0;
  int32_t cut = 0;
  const unsigned long long want = (unsigned long long)n_tokens;
  if (want < all) {
    uint32_t lo = 0, hi = 0xFFFFFFFFu;  // count(stamp < lo) <= want < count(stamp < hi)
    while (hi - lo > 1) {
      const uint32_t mid = lo + (hi - lo) / 2;
      if (int rc = count(0, mid, 0, c)) return rc;
      if (c <= want) lo = mid; else hi = mid;
    }
    S = lo;
    if (int rc = count(0, S, 0, c)) return rc;
    const unsigned long long rest = want - c;
    if (rest > 0) {
      unsigned long long lo2 = 0, hi2 = ~0ull;
      while (hi2 - lo2 > 1) {
        const unsigned long long mid = lo2 + (hi2 - lo2) / 2;
        if (int rc = count(1, S, mid, c)) return rc;
        if (c <= rest) lo2 = mid; else hi2 = mid;
      }
      K = lo2;
      if (int rc = count(1, S, K, c)) return rc;
      cut = (int32_t)(rest - c);
    }
  }
  if (int rc = push_states(r, tree, tree + 1)) return rc;
  CK(p2p::launch_lru_evict(t, r->d_states + tree, order, lvl.data(), n_levels, parent, cslot, rank, end, S, K, cut, gone,
                           surv, r->num_sms, r->stream));
  r->launches += n_levels - 1;
  if (int rc = pull_states(r, tree, tree + 1)) return rc;
  CK(p2p::launch_refresh_views(r->d_states + tree, r->d_views + tree, 1, r->d_shared, r->stream));
  r->launches += 1;
  if (n_evicted) *n_evicted = (int64_t)std::min(want, all);
  return P2P_OK;
}

int p2p_hit_rate(p2p_router* r, const int32_t* match, const int64_t* offsets, int64_t B, const int32_t* peer,
                 float* out) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (B < 0) return fail(r, P2P_E_INVAL, "negative B");
  if (B == 0) return P2P_OK;
  if (!match || !offsets || !peer || !out) return fail(r, P2P_E_INVAL, "NULL device pointer");
  DeviceGuard g(r);
  CK(p2p::launch_hit_rate(match, r->P, offsets, B, peer, out, r->num_sms, r->stream));
  r->launches += 1;
  return P2P_OK;
}

int p2p_route_prepare(p2p_router* r, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets, int64_t B) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (B < 0 || n_tokens < 0 || B > kMaxBatch) return fail(r, P2P_E_INVAL, "B or n_tokens out of range");
  if (B > 0 && (!offsets || (n_tokens > 0 && !tokens))) return fail(r, P2P_E_INVAL, "NULL device pointer");
  DeviceGuard g(r);
  if (r->prep.state == 2) CK(cudaStreamWaitEvent(r->stream, r->grp_done, 0));  // the scratch is free again
  r->prep.state = 0;
  if (B == 0) return P2P_OK;
  r->prep.tokens = tokens;
  r->prep.offsets = offsets;
  r->prep.n_tokens = n_tokens;
  r->prep.B = B;
  r->prep.state = 1;
  return P2P_OK;
}

int p2p_route_batch(p2p_router* r, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets, int64_t B,
                    const int32_t* load, int32_t alpha, int32_t* out_match, int32_t* out_peer) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (B < 0 || n_tokens < 0) return fail(r, P2P_E_INVAL, "negative B or n_tokens");
  if (B > kMaxBatch) return fail(r, P2P_E_INVAL, "B exceeds 2^30 requests per call: split the batch");
  if (int rc = check_load(r, load, alpha)) return rc;
  if (B == 0) return P2P_OK;
  if (!offsets || !out_match || !out_peer || (n_tokens > 0 && !tokens)) return fail(r, P2P_E_INVAL, "NULL device pointer");
  DeviceGuard g(r);
  if (int rc = stage_load(r, load)) return rc;
  return route(r, tokens, n_tokens, 0, offsets, B, alpha, out_match, out_peer);
}

int p2p_route_batch_decide(p2p_router* r, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets, int64_t B,
                           const int32_t* load, int32_t alpha, const uint8_t* excluded, int32_t* out_match,
                           int32_t* out_peer, int32_t* out_next) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (B < 0 || n_tokens < 0) return fail(r, P2P_E_INVAL, "negative B or n_tokens");
  if (B > kMaxBatch) return fail(r, P2P_E_INVAL, "B exceeds 2^30 requests per call: split the batch");
  if (int rc = check_load(r, load, alpha)) return rc;
  if (B == 0) return P2P_OK;
  if (!offsets || !out_match || !out_peer || (n_tokens > 0 && !tokens)) return fail(r, P2P_E_INVAL, "NULL device pointer");
  DeviceGuard g(r);
  if (int rc = stage_load(r, load, excluded)) return rc;
  return route(r, tokens, n_tokens, 0, offsets, B, alpha, out_match, out_peer, excluded != nullptr, out_next);
}

int p2p_route_decide(p2p_router* r, const int32_t* match, int64_t B, const int32_t* load, int32_t alpha,
                     const uint8_t* excluded, int32_t* out_peer, int32_t* out_next) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (B < 0) return fail(r, P2P_E_INVAL, "negative B");
  if (int rc = check_load(r, load, alpha)) return rc;
  if (B == 0) return P2P_OK;
  if (!match || !out_peer || !out_next) return fail(r, P2P_E_INVAL, "NULL device pointer");
  DeviceGuard g(r);
  if (int rc = stage_load(r, load, excluded)) return rc;
  CK(p2p::launch_decide(match, B, r->P, r->d_load, alpha, out_peer, out_next,
                        r->num_sms, r->stream));
  r->launches += 1;
  return P2P_OK;
}

int p2p_route_batch_host(p2p_router* r, const int32_t* tokens, const int64_t* offsets, int64_t B, const int32_t* load,
                         int32_t alpha, int32_t* out_match, int32_t* out_peer) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (B < 0) return fail(r, P2P_E_INVAL, "negative B");
  if (B > kMaxBatch) return fail(r, P2P_E_INVAL, "B exceeds 2^30 requests per call: split the batch");
  if (int rc = check_load(r, load, alpha)) return rc;
  if (B == 0) return P2P_OK;
  if (!offsets || !out_match || !out_peer) return fail(r, P2P_E_INVAL, "NULL host pointer");
  if (offsets[0] < 0) return fail(r, P2P_E_INVAL, "offsets[0] < 0");
  for (int64_t b = 0; b < B; ++b)
    if (offsets[b + 1] < offsets[b]) return fail(r, P2P_E_INVAL, "offsets decrease at " + std::to_string(b));
  const int64_t n_tok = offsets[B] - offsets[0];
  if (n_tok > 0 && !tokens) return fail(r, P2P_E_INVAL, "tokens is NULL");
  DeviceGuard g(r);
  CK(ensure(r, r->req_tok, (size_t)std::max<int64_t>(n_tok, 1) * sizeof(int32_t)));
  CK(ensure(r, r->req_off, (size_t)(B + 1) * sizeof(int64_t)));
  CK(ensure(r, r->out_match, (size_t)B * r->P * sizeof(int32_t)));
  CK(ensure(r, r->out_peer, (size_t)B * sizeof(int32_t)));
  if (int rc = stage_load(r, load)) return rc;
  // The batch goes in chunks: chunk k's inputs are copied in on cp_in while chunk k-1 is routed on the
  // router stream and chunk k-2's results are copied out on cp_out.  Each chunk is grouped and routed on
  // its own (groups never span chunks), which gives the same results as one pass.
  const int K = (int)std::min<int64_t>(kPipe, std::max<int64_t>(1, B / kPipeRequests));
  const int64_t Bc = (B + K - 1) / K;
  int32_t* d_tok = static_cast<int32_t*>(r->req_tok.p);
  int64_t* d_off = static_cast<int64_t*>(r->req_off.p);
  int32_t* d_match = static_cast<int32_t*>(r->out_match.p);
  int32_t* d_peer = static_cast<int32_t*>(r->out_peer.p);
  CK(cudaEventRecord(r->ev_start, r->stream));  // the buffers are ready (allocated, no longer in use)
  CK(cudaStreamWaitEvent(r->cp_in, r->ev_start, 0));
  CK(cudaStreamWaitEvent(r->cp_out, r->ev_start, 0));
  for (int k = 0; k < K; ++k) {
    const int64_t b0 = k * Bc, b1 = std::min(B, b0 + Bc);
    if (b0 >= b1) break;
    const int64_t t0 = offsets[b0] - offsets[0], t1 = offsets[b1] - offsets[0];
    if (t1 > t0)
      CK(cudaMemcpyAsync(d_tok + t0, tokens + offsets[b0], (size_t)(t1 - t0) * sizeof(int32_t), cudaMemcpyHostToDevice,
                         r->cp_in));
    CK(cudaMemcpyAsync(d_off + b0, offsets + b0, (size_t)(b1 - b0 + 1) * sizeof(int64_t), cudaMemcpyHostToDevice,
                       r->cp_in));
    CK(cudaEventRecord(r->ev_in[k], r->cp_in));
    CK(cudaStreamWaitEvent(r->stream, r->ev_in[k], 0));
    if (int rc = route(r, d_tok + t0, t1 - t0, offsets[b0], d_off + b0, b1 - b0, alpha, d_match + b0 * r->P, d_peer + b0))
      return rc;
    CK(cudaEventRecord(r->ev_routed[k], r->stream));
    CK(cudaStreamWaitEvent(r->cp_out, r->ev_routed[k], 0));
    CK(cudaMemcpyAsync(out_match + b0 * r->P, d_match + b0 * r->P, (size_t)(b1 - b0) * r->P * sizeof(int32_t),
                       cudaMemcpyDeviceToHost, r->cp_out));
    CK(cudaMemcpyAsync(out_peer + b0, d_peer + b0, (size_t)(b1 - b0) * sizeof(int32_t), cudaMemcpyDeviceToHost, r->cp_out));
  }
  CK(cudaEventRecord(r->ev_done, r->cp_out));
  CK(cudaStreamWaitEvent(r->stream, r->ev_done, 0));
  return do_sync(r);
}

}  // extern "C"
