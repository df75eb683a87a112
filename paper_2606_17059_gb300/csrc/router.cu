// router.cu -- host runtime of the routing engine: the C ABI declared in p2p_router.h.
//
// The router owns P trees in HBM (layout in internal.h), allocated from a router-private stream-ordered
// memory pool so that replacing a tree (snapshot upload, arena growth) frees the old arrays in stream
// order, after any route still reading them.  All device work goes to the router's stream.
#include <algorithm>
#include <cstring>
#include <string>
#include <vector>

#include "internal.h"

using p2p::TreeState;
using p2p::TreeView;

namespace {

constexpr int kLoadRing = 8;

struct DevBuf {
  void* p = nullptr;
  size_t cap = 0;
};

int32_t clamp_i32(int64_t v) { return (int32_t)std::min<int64_t>(v, INT32_MAX); }

}  // namespace

struct p2p_router {
  int32_t P = 0;
  int device = 0;
  int num_sms = 0;
  cudaStream_t stream = nullptr;
  cudaMemPool_t pool = nullptr;
  std::vector<TreeState> hs;  // host mirror of every tree's state
  TreeView* d_views = nullptr;
  TreeState* d_states = nullptr;
  int32_t* d_load = nullptr;
  int32_t* d_err = nullptr;
  int32_t* h_load = nullptr;  // pinned, kLoadRing slots of P values
  cudaEvent_t load_ev[kLoadRing] = {};
  int load_slot = 0;
  int32_t* h_err = nullptr;        // pinned
  TreeState* h_states = nullptr;   // pinned, P entries
  DevBuf req_tok, req_off, out_match, out_peer;
  DevBuf d_op, d_seg_begin, d_seg_off, d_seg_len, d_pool, d_scratch;
  int64_t launches = 0;  // kernels this router has launched
  std::string err;
};

namespace {

// Makes the router's device current for the duration of a call.
struct DeviceGuard {
  int prev = -1;
  bool changed = false;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) changed = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
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

#define CK(call)                                         \
  do {                                                   \
    cudaError_t e_ = (call);                             \
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

// Device-to-host copy ordered on the router stream (waits for it).
cudaError_t d2h(p2p_router* r, void* dst, const void* src, size_t bytes) {
  cudaError_t e = cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToHost, r->stream);
  return e == cudaSuccess ? cudaStreamSynchronize(r->stream) : e;
}

void free_tree_arrays(p2p_router* r, TreeState& t) {
  dfree(r, t.node);
  dfree(r, t.child);
  dfree(r, t.label);
  t.node = nullptr;
  t.child = nullptr;
  t.label = nullptr;
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
  t.free_head = -1;
  return cudaSuccess;
}

int install_empty_tree(p2p_router* r, int32_t p) {
  TreeState t;
  cudaError_t e = alloc_tree_arrays(r, t, 64, 64, 1024);
  if (e != cudaSuccess) return cuda_fail(r, e, "allocating an empty tree");
  CK(cudaMemsetAsync(t.node, 0, sizeof(int4), r->stream));
  t.n_node = 1;
  r->hs[(size_t)p] = t;
  CK(p2p::launch_set_tree(r->d_states + p, r->d_views + p, t, r->stream));
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

// Stages load[P] through a pinned ring slot (the slot's previous copy has finished once its event has).
int stage_load(p2p_router* r, const int32_t* load) {
  const int s = r->load_slot;
  r->load_slot = (s + 1) % kLoadRing;
  CK(cudaEventSynchronize(r->load_ev[s]));
  int32_t* slot = r->h_load + (size_t)s * r->P;
  std::memcpy(slot, load, (size_t)r->P * sizeof(int32_t));
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
    return fail(r, P2P_E_DEVICE, m);
  }
  return P2P_OK;
}

int upload_flat(p2p_router* r, int32_t peer, const p2p_flat_tree* t) {
  std::string err;
  if (!p2p::validate_flat(t, err)) return fail(r, P2P_E_FORMAT, err);
  const int64_t N = t->n_nodes, NL = t->n_labels;
  std::vector<int4> node((size_t)N), child((size_t)std::max<int64_t>(N - 1, 0));
  for (int64_t v = 0; v < N; ++v) node[(size_t)v] = make_int4(t->child_begin[v], t->child_count[v], t->child_count[v], t->term_count[v]);
  for (int64_t e = 0; e < N - 1; ++e) {
    const int32_t c = t->child_idx[e];
    child[(size_t)e] = make_int4(t->child_first_tok[e], c, t->label_off[c], t->label_len[c]);
  }
  const int32_t cap_node = clamp_i32(N + std::max<int64_t>(N / 4, 64));
  const int32_t cap_child = clamp_i32((N - 1) + std::max<int64_t>((N - 1) / 2, 64));
  const int32_t cap_label = clamp_i32(NL + std::max<int64_t>(NL / 4, 1024));
  TreeState nt;
  cudaError_t e = alloc_tree_arrays(r, nt, cap_node, cap_child, cap_label);
  if (e != cudaSuccess) return fail(r, P2P_E_NOMEM, std::string("allocating the tree: ") + cudaGetErrorString(e));
  CK(cudaMemcpyAsync(nt.node, node.data(), (size_t)N * sizeof(int4), cudaMemcpyHostToDevice, r->stream));
  if (N > 1) CK(cudaMemcpyAsync(nt.child, child.data(), (size_t)(N - 1) * sizeof(int4), cudaMemcpyHostToDevice, r->stream));
  if (NL > 0) CK(cudaMemcpyAsync(nt.label, t->labels, (size_t)NL * sizeof(int32_t), cudaMemcpyHostToDevice, r->stream));
  nt.n_node = (int32_t)N;
  nt.n_child = (int32_t)(N - 1);
  nt.n_label = (int32_t)NL;
  TreeState& old = r->hs[(size_t)peer];
  free_tree_arrays(r, old);
  old = nt;
  CK(p2p::launch_set_tree(r->d_states + peer, r->d_views + peer, nt, r->stream));
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
  if (!p2p::snapshot_from_device_layout(node.data(), t.n_node, child.data(), t.n_child, label.data(), t.n_label, *out, err))
    return fail(r, P2P_E_DEVICE, err);
  return P2P_OK;
}

// Grows the arenas of tree p so that the op that stopped with DELTA_NEED_SPACE fits.
int grow_tree(p2p_router* r, int32_t p) {
  TreeState& t = r->hs[(size_t)p];
  const int64_t nodes_short = (int64_t)t.need_node - t.n_free - ((int64_t)t.cap_node - t.n_node);
  const int64_t child_short = (int64_t)t.need_child - ((int64_t)t.cap_child - t.n_child);
  const int64_t label_short = (int64_t)t.need_label - ((int64_t)t.cap_label - t.n_label);
  auto newcap = [](int64_t cap, int64_t used, int64_t need) -> int64_t {
    return std::max<int64_t>(cap * 2, used + 2 * need + 1024);
  };
  TreeState nt = t;
  int64_t cn = t.cap_node, cc = t.cap_child, cl = t.cap_label;
  if (nodes_short > 0) cn = newcap(t.cap_node, t.n_node, t.need_node);
  if (child_short > 0) cc = newcap(t.cap_child, t.n_child, t.need_child);
  if (label_short > 0) cl = newcap(t.cap_label, t.n_label, t.need_label);
  if ((nodes_short > 0 && (int64_t)t.n_node + t.need_node > INT32_MAX) ||
      (child_short > 0 && (int64_t)t.n_child + t.need_child > INT32_MAX) ||
      (label_short > 0 && (int64_t)t.n_label + t.need_label > INT32_MAX))
    return fail(r, P2P_E_NOMEM, "tree " + std::to_string(p) + " outgrows the int32 arena indices");
  cn = std::min<int64_t>(cn, INT32_MAX);
  cc = std::min<int64_t>(cc, INT32_MAX);
  cl = std::min<int64_t>(cl, INT32_MAX);
  int4* nn = t.node;
  int4* nc = t.child;
  int32_t* nl = t.label;
  cudaError_t e = cudaSuccess;
  if (cn != t.cap_node && e == cudaSuccess) e = dalloc(r, (void**)&nn, (size_t)cn * sizeof(int4));
  if (cc != t.cap_child && e == cudaSuccess) e = dalloc(r, (void**)&nc, (size_t)cc * sizeof(int4));
  if (cl != t.cap_label && e == cudaSuccess) e = dalloc(r, (void**)&nl, (size_t)cl * sizeof(int32_t));
  if (e != cudaSuccess) {
    if (nn != t.node) dfree(r, nn);
    if (nc != t.child) dfree(r, nc);
    if (nl != t.label) dfree(r, nl);
    return fail(r, P2P_E_NOMEM, std::string("growing a tree: ") + cudaGetErrorString(e));
  }
  if (nn != t.node) {
    CK(cudaMemcpyAsync(nn, t.node, (size_t)t.n_node * sizeof(int4), cudaMemcpyDeviceToDevice, r->stream));
    dfree(r, t.node);
  }
  if (nc != t.child) {
    CK(cudaMemcpyAsync(nc, t.child, (size_t)t.n_child * sizeof(int4), cudaMemcpyDeviceToDevice, r->stream));
    dfree(r, t.child);
  }
  if (nl != t.label) {
    CK(cudaMemcpyAsync(nl, t.label, (size_t)t.n_label * sizeof(int32_t), cudaMemcpyDeviceToDevice, r->stream));
    dfree(r, t.label);
  }
  nt.node = nn;
  nt.child = nc;
  nt.label = nl;
  nt.cap_node = (int32_t)cn;
  nt.cap_child = (int32_t)cc;
  nt.cap_label = (int32_t)cl;
  nt.status = p2p::DELTA_OK;
  t = nt;
  return P2P_OK;
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
  e = dalloc(r, (void**)&r->d_views, (size_t)P * sizeof(TreeView));
  if (e == cudaSuccess) e = dalloc(r, (void**)&r->d_states, (size_t)P * sizeof(TreeState));
  if (e == cudaSuccess) e = dalloc(r, (void**)&r->d_load, (size_t)P * sizeof(int32_t));
  if (e == cudaSuccess) e = dalloc(r, (void**)&r->d_err, sizeof(int32_t));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&r->h_load, (size_t)kLoadRing * P * sizeof(int32_t));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&r->h_err, sizeof(int32_t));
  if (e == cudaSuccess) e = cudaMallocHost((void**)&r->h_states, (size_t)P * sizeof(TreeState));
  for (int i = 0; i < kLoadRing && e == cudaSuccess; ++i) e = cudaEventCreateWithFlags(&r->load_ev[i], cudaEventDisableTiming);
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
  DeviceGuard g(r->device);
  cudaStreamSynchronize(r->stream);
  if (r->pool) {
    for (TreeState& t : r->hs) free_tree_arrays(r, t);
    for (DevBuf* b : {&r->req_tok, &r->req_off, &r->out_match, &r->out_peer, &r->d_op, &r->d_seg_begin,
                      &r->d_seg_off, &r->d_seg_len, &r->d_pool, &r->d_scratch})
      dfree(r, b->p);
    dfree(r, r->d_views);
    dfree(r, r->d_states);
    dfree(r, r->d_load);
    dfree(r, r->d_err);
    cudaStreamSynchronize(r->stream);
    cudaMemPoolDestroy(r->pool);
  }
  for (cudaEvent_t ev : r->load_ev)
    if (ev) cudaEventDestroy(ev);
  if (r->h_load) cudaFreeHost(r->h_load);
  if (r->h_err) cudaFreeHost(r->h_err);
  if (r->h_states) cudaFreeHost(r->h_states);
  delete r;
}

int p2p_router_set_stream(p2p_router* r, void* stream) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  DeviceGuard g(r->device);
  CK(cudaStreamSynchronize(r->stream));
  r->stream = (cudaStream_t)stream;
  return P2P_OK;
}

int p2p_router_sync(p2p_router* r) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  DeviceGuard g(r->device);
  return do_sync(r);
}

const char* p2p_last_error(const p2p_router* r) { return r ? r->err.c_str() : p2p::global_error(); }

int32_t p2p_router_num_trees(const p2p_router* r) { return r ? r->P : 0; }

int64_t p2p_router_launch_count(const p2p_router* r) { return r ? r->launches : 0; }

int p2p_tree_upload(p2p_router* r, int32_t peer, const p2p_flat_tree* t) {
  if (int rc = check_peer(r, peer)) return rc;
  DeviceGuard g(r->device);
  return upload_flat(r, peer, t);
}

int p2p_tree_build(p2p_router* r, int32_t peer, const p2p_seqs* seqs) {
  if (int rc = check_peer(r, peer)) return rc;
  std::string err;
  if (!seqs || !p2p::check_seqs(seqs, err, nullptr, nullptr)) return fail(r, P2P_E_INVAL, seqs ? err : "seqs is NULL");
  p2p_snapshot snap;
  if (!p2p::build_snapshot(*seqs, snap, err)) return fail(r, P2P_E_NOMEM, err);
  p2p_flat_tree v;
  p2p_snapshot_view(&snap, &v);
  DeviceGuard g(r->device);
  return upload_flat(r, peer, &v);
}

int p2p_tree_download(p2p_router* r, int32_t peer, p2p_snapshot** out) {
  if (int rc = check_peer(r, peer)) return rc;
  if (!out) return fail(r, P2P_E_INVAL, "out is NULL");
  *out = nullptr;
  DeviceGuard g(r->device);
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
  DeviceGuard g(r->device);
  CK(cudaStreamSynchronize(r->stream));
  const TreeState& t = r->hs[(size_t)peer];
  const int64_t v[9] = {(int64_t)t.n_node - t.n_free, t.n_node, t.n_child, t.n_label, t.stale_child,
                        t.stale_label, t.cap_node, t.cap_child, t.cap_label};
  std::memcpy(out, v, sizeof(v));
  return P2P_OK;
}

int p2p_tree_apply_delta(p2p_router* r, int32_t peer, const p2p_delta* d, int64_t* n_absent) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (peer < -1 || peer >= r->P) return fail(r, P2P_E_INVAL, "peer out of range");
  if (!d) return fail(r, P2P_E_INVAL, "delta is NULL");
  if (d->mem != P2P_MEM_HOST && d->mem != P2P_MEM_DEVICE) return fail(r, P2P_E_INVAL, "delta.mem must be HOST or DEVICE");
  DeviceGuard g(r->device);
  const p2p_seqs& S = d->seqs;
  const int64_t n = S.n;
  if (n < 0 || S.n_segs < 0 || S.n_pool < 0) return fail(r, P2P_E_INVAL, "negative size in delta");
  if (n > 0 && (!d->op || !S.seg_begin)) return fail(r, P2P_E_INVAL, "NULL op or seg_begin");
  // Host view of the op metadata (device deltas: copy it out to validate it; the pool stays on the device).
  std::vector<int32_t> h_op, h_seg_len;
  std::vector<int64_t> h_seg_begin, h_seg_off, h_peer_begin;
  const int32_t* op = d->op;
  const int64_t* peer_begin = d->peer_begin;
  p2p_seqs hv = S;
  if (d->mem == P2P_MEM_DEVICE) {
    CK(cudaStreamSynchronize(r->stream));
    h_op.resize((size_t)n);
    h_seg_begin.resize((size_t)n + 1);
    h_seg_off.resize((size_t)S.n_segs);
    h_seg_len.resize((size_t)S.n_segs);
    if (n) CK(d2h(r, h_op.data(), d->op, (size_t)n * sizeof(int32_t)));
    if (S.seg_begin) CK(d2h(r, h_seg_begin.data(), S.seg_begin, (size_t)(n + 1) * sizeof(int64_t)));
    if (S.n_segs && S.seg_off && S.seg_len) {
      CK(d2h(r, h_seg_off.data(), S.seg_off, (size_t)S.n_segs * sizeof(int64_t)));
      CK(d2h(r, h_seg_len.data(), S.seg_len, (size_t)S.n_segs * sizeof(int32_t)));
    }
    if (peer == -1 && d->peer_begin) {
      h_peer_begin.resize((size_t)r->P + 1);
      CK(d2h(r, h_peer_begin.data(), d->peer_begin, (size_t)(r->P + 1) * sizeof(int64_t)));
      peer_begin = h_peer_begin.data();
    }
    op = h_op.data();
    hv.seg_begin = S.seg_begin ? h_seg_begin.data() : nullptr;
    hv.seg_off = S.seg_off ? h_seg_off.data() : nullptr;
    hv.seg_len = S.seg_len ? h_seg_len.data() : nullptr;
  }
  if (n == 0) {
    if (n_absent) *n_absent = 0;
    return P2P_OK;
  }
  std::string err;
  int64_t max_len = 0;
  if (!p2p::check_seqs(&hv, err, &max_len, nullptr)) return fail(r, P2P_E_INVAL, err);
  for (int64_t i = 0; i < n; ++i)
    if (op[i] != P2P_OP_INSERT && op[i] != P2P_OP_DELETE) return fail(r, P2P_E_INVAL, "bad op code at " + std::to_string(i));
  if (peer == -1) {
    if (!peer_begin) return fail(r, P2P_E_INVAL, "peer = -1 needs peer_begin");
    if (peer_begin[0] != 0 || peer_begin[r->P] != n) return fail(r, P2P_E_INVAL, "peer_begin must run from 0 to n");
    for (int32_t p = 0; p < r->P; ++p)
      if (peer_begin[p + 1] < peer_begin[p]) return fail(r, P2P_E_INVAL, "peer_begin not non-decreasing");
  }
  // Device copies of the delta.
  const int32_t* d_op = d->op;
  const int64_t *d_sb = S.seg_begin, *d_so = S.seg_off;
  const int32_t *d_sl = S.seg_len, *d_pool = S.pool;
  if (d->mem == P2P_MEM_HOST) {
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
    d_op = (const int32_t*)r->d_op.p;
    d_sb = (const int64_t*)r->d_seg_begin.p;
    d_so = (const int64_t*)r->d_seg_off.p;
    d_sl = (const int32_t*)r->d_seg_len.p;
    d_pool = (const int32_t*)r->d_pool.p;
  }
  // Trees touched by this call and their op ranges.
  const int32_t p0 = peer == -1 ? 0 : peer, p1 = peer == -1 ? r->P : peer + 1;
  for (int32_t p = p0; p < p1; ++p) {
    TreeState& t = r->hs[(size_t)p];
    t.op_next = peer == -1 ? peer_begin[p] : 0;
    t.op_end = peer == -1 ? peer_begin[p + 1] : n;
    t.status = p2p::DELTA_OK;
    t.n_absent = 0;
  }
  const int32_t nt = p1 - p0;
  const int64_t stride = std::max<int64_t>(max_len, 1);
  CK(ensure(r, r->d_scratch, (size_t)nt * stride * sizeof(int32_t)));
  int rc = P2P_OK;
  for (int round = 0;; ++round) {
    std::memcpy(r->h_states, r->hs.data() + p0, (size_t)nt * sizeof(TreeState));
    CK(cudaMemcpyAsync(r->d_states + p0, r->h_states, (size_t)nt * sizeof(TreeState), cudaMemcpyHostToDevice, r->stream));
    CK(p2p::launch_delta(r->d_states + p0, nt, d_op, d_sb, d_so, d_sl, d_pool, (int32_t*)r->d_scratch.p, stride, r->stream));
    r->launches += 1;
    CK(cudaMemcpyAsync(r->h_states, r->d_states + p0, (size_t)nt * sizeof(TreeState), cudaMemcpyDeviceToHost, r->stream));
    CK(cudaStreamSynchronize(r->stream));
    std::memcpy(r->hs.data() + p0, r->h_states, (size_t)nt * sizeof(TreeState));
    bool again = false;
    for (int32_t p = p0; p < p1 && rc == P2P_OK; ++p) {
      TreeState& t = r->hs[(size_t)p];
      if (t.status == p2p::DELTA_CORRUPT) {
        rc = fail(r, P2P_E_DEVICE, "tree " + std::to_string(p) + " is inconsistent (delta stopped at op " + std::to_string(t.op_next) + ")");
      } else if (t.status == p2p::DELTA_NEED_SPACE) {
        rc = grow_tree(r, p);
        again = true;
      }
    }
    if (rc != P2P_OK || !again) break;
  }
  // Publish the (possibly moved) arrays to the route kernel's view table; compact very stale trees.
  std::memcpy(r->h_states, r->hs.data() + p0, (size_t)nt * sizeof(TreeState));
  CK(cudaMemcpyAsync(r->d_states + p0, r->h_states, (size_t)nt * sizeof(TreeState), cudaMemcpyHostToDevice, r->stream));
  CK(p2p::launch_refresh_views(r->d_states + p0, r->d_views + p0, nt, r->stream));
  r->launches += 1;
  int64_t absent = 0;
  for (int32_t p = p0; p < p1; ++p) {
    TreeState& t = r->hs[(size_t)p];
    absent += t.n_absent;
    const int64_t used = (int64_t)t.n_child + t.n_label;
    const int64_t stale = t.stale_child + t.stale_label;
    if (rc == P2P_OK && stale > 65536 && 2 * stale > used) rc = compact_tree(r, p);
  }
  // h_states is reused by the next call only after this copy has run.
  CK(cudaStreamSynchronize(r->stream));
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
  DeviceGuard g(r->device);
  int32_t* header = nullptr;
  int32_t* tokens = nullptr;
  CK(p2p::static_scratch(r->device, &header, &tokens));
  if (S.n == 0) {
    if (n_absent) *n_absent = 0;
    return P2P_OK;
  }
  CK(p2p::launch_validate_static(header, d, peer, r->P, r->stream));
  r->launches += 1;
  int32_t h[4] = {0, 0, 0, 0};
  CK(cudaMemcpyAsync(h, header, sizeof(h), cudaMemcpyDeviceToHost, r->stream));
  CK(cudaStreamSynchronize(r->stream));
  unsigned long long max_len = 0;
  std::memcpy(&max_len, h, sizeof(max_len));
  const int32_t bits = h[2];
  if (bits & p2p::STATIC_BAD_OP) return fail(r, P2P_E_INVAL, "bad op code in the delta");
  if (bits & p2p::STATIC_BAD_SEGMENT) return fail(r, P2P_E_INVAL, "seg_begin or a segment is malformed or outside the pool");
  if (bits & p2p::STATIC_TOO_LONG) return fail(r, P2P_E_INVAL, "a sequence is longer than 2^31-1 tokens");
  if (bits & p2p::STATIC_BAD_PEER_BEGIN) return fail(r, P2P_E_INVAL, "peer_begin must run non-decreasing from 0 to n");
  const int32_t p0 = peer == -1 ? 0 : peer, p1 = peer == -1 ? r->P : peer + 1;
  const int32_t nt = p1 - p0;
  const int64_t stride = max_len > 0 ? (int64_t)max_len : 1;
  if ((int64_t)nt * stride > p2p::static_scratch_tokens())
    return fail(r, P2P_E_INVAL, "trees x longest sequence = " + std::to_string((int64_t)nt * stride) +
                                    " tokens exceeds the static scratch of " +
                                    std::to_string(p2p::static_scratch_tokens()) + " tokens");
  CK(p2p::launch_init_ranges(r->d_states + p0, nt, peer == -1 ? d->peer_begin : nullptr, S.n, r->stream));
  CK(p2p::launch_delta(r->d_states + p0, nt, d->op, S.seg_begin, S.seg_off, S.seg_len, S.pool, tokens, stride, r->stream));
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
    if (t.status == p2p::DELTA_CORRUPT)
      rc = fail(r, P2P_E_DEVICE, "tree " + std::to_string(p) + " is inconsistent (delta stopped at op " + std::to_string(t.op_next) + ")");
    else if (t.status == p2p::DELTA_NEED_SPACE)
      rc = fail(r, P2P_E_NOMEM, "tree " + std::to_string(p) + " has no room for op " + std::to_string(t.op_next) +
                                    "; its earlier ops were applied (p2p_tree_apply_delta grows trees)");
  }
  if (n_absent) *n_absent = absent;
  return rc;
}

int p2p_route_batch(p2p_router* r, const int32_t* tokens, int64_t n_tokens, const int64_t* offsets, int64_t B,
                    const int32_t* load, int32_t alpha, int32_t* out_match, int32_t* out_peer) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (B < 0 || n_tokens < 0) return fail(r, P2P_E_INVAL, "negative B or n_tokens");
  if (int rc = check_load(r, load, alpha)) return rc;
  if (B == 0) return P2P_OK;
  if (!offsets || !out_match || !out_peer || (n_tokens > 0 && !tokens)) return fail(r, P2P_E_INVAL, "NULL device pointer");
  DeviceGuard g(r->device);
  if (int rc = stage_load(r, load)) return rc;
  CK(p2p::launch_route(r->d_views, r->P, tokens, n_tokens, 0, offsets, B, r->d_load, alpha, out_match, out_peer,
                       r->d_err, r->num_sms, r->stream));
  r->launches += 1;
  return P2P_OK;
}

int p2p_route_batch_host(p2p_router* r, const int32_t* tokens, const int64_t* offsets, int64_t B, const int32_t* load,
                         int32_t alpha, int32_t* out_match, int32_t* out_peer) {
  if (!r) return fail(nullptr, P2P_E_INVAL, "router is NULL");
  if (B < 0) return fail(r, P2P_E_INVAL, "negative B");
  if (int rc = check_load(r, load, alpha)) return rc;
  if (B == 0) return P2P_OK;
  if (!offsets || !out_match || !out_peer) return fail(r, P2P_E_INVAL, "NULL host pointer");
  if (offsets[0] < 0) return fail(r, P2P_E_INVAL, "offsets[0] < 0");
  for (int64_t b = 0; b < B; ++b)
    if (offsets[b + 1] < offsets[b]) return fail(r, P2P_E_INVAL, "offsets decrease at " + std::to_string(b));
  const int64_t n_tok = offsets[B] - offsets[0];
  if (n_tok > 0 && !tokens) return fail(r, P2P_E_INVAL, "tokens is NULL");
  DeviceGuard g(r->device);
  CK(ensure(r, r->req_tok, (size_t)std::max<int64_t>(n_tok, 1) * sizeof(int32_t)));
  CK(ensure(r, r->req_off, (size_t)(B + 1) * sizeof(int64_t)));
  CK(ensure(r, r->out_match, (size_t)B * r->P * sizeof(int32_t)));
  CK(ensure(r, r->out_peer, (size_t)B * sizeof(int32_t)));
  if (n_tok) CK(cudaMemcpyAsync(r->req_tok.p, tokens + offsets[0], (size_t)n_tok * sizeof(int32_t), cudaMemcpyHostToDevice, r->stream));
  CK(cudaMemcpyAsync(r->req_off.p, offsets, (size_t)(B + 1) * sizeof(int64_t), cudaMemcpyHostToDevice, r->stream));
  if (int rc = stage_load(r, load)) return rc;
  CK(p2p::launch_route(r->d_views, r->P, (const int32_t*)r->req_tok.p, n_tok, offsets[0], (const int64_t*)r->req_off.p, B,
                       r->d_load, alpha, (int32_t*)r->out_match.p, (int32_t*)r->out_peer.p, r->d_err, r->num_sms,
                       r->stream));
  r->launches += 1;
  CK(cudaMemcpyAsync(out_match, r->out_match.p, (size_t)B * r->P * sizeof(int32_t), cudaMemcpyDeviceToHost, r->stream));
  CK(cudaMemcpyAsync(out_peer, r->out_peer.p, (size_t)B * sizeof(int32_t), cudaMemcpyDeviceToHost, r->stream));
  return do_sync(r);
}

}  // extern "C"
