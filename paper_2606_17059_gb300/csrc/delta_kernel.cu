// delta_kernel.cu -- anti-entropy delta applied to radix-tree replicas in HBM.
//
// An ordered list of ops patches one or more trees: INSERT adds one occurrence of a token sequence
// (updateTrie / updateTrieEstimate in the paper's Section 2 primitive list), DELETE removes one (a
// counted no-op when the sequence is not stored).  Trees stay edge-compressed and canonical: an INSERT
// that leaves an edge part-way splits it; a DELETE prunes a leaf that no longer stores anything and folds
// a node left with one child and no sequence into that child.
//
// Mapping: one warp per tree; a tree's ops run in order, trees run in parallel.  Inside an op the warp
// cooperates: the sequence is gathered into a per-warp scratch run, child searches probe 32 sorted first
// tokens at a time, label compares and copies move 32 tokens per instruction, child-list shifts move 32
// entries per step.  Lane 0 performs the scalar stores; __syncwarp() orders them before the next reads.
// Before mutating, an op checks that the node, child-entry and label arenas have room for everything it
// may allocate; if not, the tree stops at that op with DELTA_NEED_SPACE and the host grows the arenas and
// relaunches, so every op is applied whole or not at all.  All loops are bounded by sequence lengths
// and list sizes.
#include "internal.h"

namespace p2p {
namespace {

constexpr unsigned kFull = 0xffffffffu;
enum { OP_DONE = 0, OP_NEED = 1, OP_CORRUPT = 2 };

// Index of `tok` among child entries [b, b + cnt) (sorted by .x), or the slot where it would go.
__device__ bool search(const int4* child, int32_t b, int32_t cnt, int32_t tok, int lane, int32_t& at) {
  int32_t lo = b, hi = b + cnt;
  while (hi - lo > 32) {
    const int32_t step = (hi - lo + 31) >> 5;
    const int32_t idx = lo + lane * step;
    const bool le = idx < hi && child[idx].x <= tok;
    const int c = __popc(__ballot_sync(kFull, le));
    if (c == 0) {
      at = lo;
      return false;
    }
    lo += (c - 1) * step;
    hi = min(lo + step, hi);
  }
  const bool valid = lo + lane < hi;
  const int32_t key = valid ? child[lo + lane].x : 0;
  const unsigned lt = __ballot_sync(kFull, valid && key < tok);
  const unsigned eq = __ballot_sync(kFull, valid && key == tok);
  at = lo + __popc(lt);
  return eq != 0;
}

// First j in [from, lim) with a[j] != b[j], or lim.
__device__ int64_t first_diff(const int32_t* a, const int32_t* b, int64_t from, int64_t lim, int lane) {
  for (int64_t j0 = from; j0 < lim; j0 += 128) {
    int32_t x[4], y[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t j = j0 + u * 32 + lane;
      x[u] = j < lim ? a[j] : 0;
      y[u] = j < lim ? b[j] : 0;
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const unsigned m = __ballot_sync(kFull, x[u] != y[u]);
      if (m) return j0 + u * 32 + (__ffs(m) - 1);
    }
  }
  return lim;
}

__device__ void copy_tokens(int32_t* dst, const int32_t* src, int64_t n, int lane) {
  for (int64_t j = lane; j < n; j += 32) dst[j] = src[j];
}

// Moves child entries [lo, hi) up by one slot (top chunk first, so nothing is overwritten unread).
__device__ void shift_up(int4* child, int64_t lo, int64_t hi, int lane) {
  for (int64_t top = hi; top > lo; top -= 32) {
    const int64_t base = top - 32 > lo ? top - 32 : lo;
    const int64_t j = base + lane;
    int4 v = make_int4(0, 0, 0, 0);
    if (j < top) v = child[j];
    __syncwarp();
    if (j < top) child[j + 1] = v;
    __syncwarp();
  }
}

// Moves child entries [lo, hi) down by one slot (bottom chunk first).
__device__ void shift_down(int4* child, int64_t lo, int64_t hi, int lane) {
  for (int64_t base = lo; base < hi; base += 32) {
    const int64_t j = base + lane;
    int4 v = make_int4(0, 0, 0, 0);
    if (j < hi) v = child[j];
    __syncwarp();
    if (j < hi) child[j - 1] = v;
    __syncwarp();
  }
}

__device__ bool has_room(TreeState& s, int64_t nodes, int64_t entries, int64_t tokens) {
  if ((int64_t)s.n_free + ((int64_t)s.cap_node - s.n_node) >= nodes && (int64_t)s.cap_child - s.n_child >= entries &&
      (int64_t)s.cap_label - s.n_label >= tokens)
    return true;
  s.need_node = (int32_t)nodes;
  s.need_child = (int32_t)entries;
  s.need_label = (int32_t)(tokens > INT32_MAX ? INT32_MAX : tokens);
  return false;
}

__device__ int32_t alloc_node(TreeState& s) {
  if (s.free_head >= 0) {
    const int32_t v = s.free_head;
    s.free_head = s.node[v].x;
    s.n_free -= 1;
    return v;
  }
  return s.n_node++;
}

__device__ void free_node(TreeState& s, int32_t v, int lane) {
  if (lane == 0) s.node[v] = make_int4(s.free_head, 0, 0, 0);
  s.free_head = v;
  s.n_free += 1;
}

// Node x (reached through parent entry ex) has one child and stores no sequence: fold the child into x.
// The caller has checked that the label arena has room for the two labels.
__device__ void merge_into_parent(TreeState& s, int32_t x, int32_t ex, int lane) {
  const int4 xe = s.child[ex];
  const int4 xn = s.node[x];
  const int4 ye = s.child[xn.x];
  const int4 yn = s.node[ye.y];
  int32_t off = xe.z;
  if (xe.z + xe.w != ye.z) {  // labels not adjacent in the arena: write the joined label
    off = s.n_label;
    copy_tokens(s.label + off, s.label + xe.z, xe.w, lane);
    copy_tokens(s.label + off + xe.w, s.label + ye.z, ye.w, lane);
    s.n_label += xe.w + ye.w;
    s.stale_label += xe.w + ye.w;
  }
  __syncwarp();
  if (lane == 0) {
    s.child[ex] = make_int4(xe.x, x, off, xe.w + ye.w);
    s.node[x] = yn;
  }
  s.stale_child += xn.z;
  free_node(s, ye.y, lane);
  __syncwarp();
}

__device__ bool adjacent_labels(const TreeState& s, int32_t ex, int32_t ey) {
  const int4 a = s.child[ex], b = s.child[ey];
  return a.z + a.w == b.z;
}

__device__ int insert(TreeState& s, const int32_t* seq, int64_t n, int lane) {
  int32_t cur = 0;
  int64_t pos = 0;
  for (int64_t guard = 0; guard <= n + 1; ++guard) {
    const int4 nd = s.node[cur];
    if (pos == n) {
      if (lane == 0) s.node[cur].w = nd.w + 1;
      __syncwarp();
      return OP_DONE;
    }
    const int32_t tok = seq[pos];
    int32_t at;
    if (!search(s.child, nd.x, nd.y, tok, lane, at)) {
      // New leaf edge seq[pos, n) under cur, at slot `at` of cur's (sorted) child list.
      const int64_t L = n - pos;
      const bool grow = nd.y >= nd.z;
      const int32_t newcap = grow ? max(2, 2 * nd.y) : 0;
      if (!has_room(s, 1, newcap, L)) return OP_NEED;
      const int32_t leaf = alloc_node(s);
      const int32_t loff = s.n_label;
      copy_tokens(s.label + loff, seq + pos, L, lane);
      s.n_label += (int32_t)L;
      const int4 ent = make_int4(tok, leaf, loff, (int32_t)L);
      if (!grow) {
        shift_up(s.child, at, (int64_t)nd.x + nd.y, lane);
        if (lane == 0) {
          s.child[at] = ent;
          s.node[cur].y = nd.y + 1;
        }
      } else {
        const int32_t nb = s.n_child;
        s.n_child += newcap;
        const int32_t before = at - nd.x;
        for (int64_t j = lane; j < nd.y; j += 32) {
          const int4 v = s.child[nd.x + j];
          s.child[nb + j + (j >= before ? 1 : 0)] = v;
        }
        if (lane == 0) {
          s.child[nb + before] = ent;
          s.node[cur] = make_int4(nb, nd.y + 1, newcap, nd.w);
        }
        s.stale_child += nd.z;
      }
      if (lane == 0) s.node[leaf] = make_int4(0, 0, 0, 1);
      __syncwarp();
      return OP_DONE;
    }
    const int4 ce = s.child[at];
    if (ce.w <= 0 || ce.y <= 0) return OP_CORRUPT;
    const int64_t lim = min((int64_t)ce.w, n - pos);
    const int64_t k = first_diff(s.label + ce.z, seq + pos, 1, lim, lane);
    if (k == ce.w) {
      cur = ce.y;
      pos += k;
      continue;
    }
    // The sequence leaves (or ends inside) the edge after k tokens: split it there.
    const bool tail = pos + k < n;
    const int64_t L = n - pos - k;
    if (!has_room(s, tail ? 2 : 1, 2, tail ? L : 0)) return OP_NEED;
    const int32_t mid = alloc_node(s);
    const int32_t leaf = tail ? alloc_node(s) : -1;
    const int32_t nb = s.n_child;
    s.n_child += 2;
    const int4 lower = make_int4(s.label[ce.z + k], ce.y, ce.z + (int32_t)k, ce.w - (int32_t)k);
    int4 leaf_ent = make_int4(0, 0, 0, 0);
    if (tail) {
      const int32_t loff = s.n_label;
      copy_tokens(s.label + loff, seq + pos + k, L, lane);
      s.n_label += (int32_t)L;
      leaf_ent = make_int4(seq[pos + k], leaf, loff, (int32_t)L);
    }
    if (lane == 0) {
      if (tail) {
        const bool leaf_first = leaf_ent.x < lower.x;
        s.child[nb] = leaf_first ? leaf_ent : lower;
        s.child[nb + 1] = leaf_first ? lower : leaf_ent;
        s.node[leaf] = make_int4(0, 0, 0, 1);
      } else {
        s.child[nb] = lower;
      }
      s.node[mid] = make_int4(nb, tail ? 2 : 1, 2, tail ? 0 : 1);
      s.child[at] = make_int4(ce.x, mid, ce.z, (int32_t)k);
    }
    __syncwarp();
    return OP_DONE;
  }
  return OP_CORRUPT;
}

__device__ int remove(TreeState& s, const int32_t* seq, int64_t n, int lane) {
  int32_t cur = 0, par = -1, e_cur = -1, e_par = -1;
  int64_t pos = 0;
  for (int64_t guard = 0; pos < n; ++guard) {
    if (guard > n) return OP_CORRUPT;
    const int4 nd = s.node[cur];
    int32_t at;
    if (!search(s.child, nd.x, nd.y, seq[pos], lane, at)) {
      s.n_absent += 1;
      return OP_DONE;
    }
    const int4 ce = s.child[at];
    if (ce.w <= 0 || ce.y <= 0) return OP_CORRUPT;
    if (pos + ce.w > n || first_diff(s.label + ce.z, seq + pos, 1, ce.w, lane) < ce.w) {
      s.n_absent += 1;
      return OP_DONE;
    }
    e_par = e_cur;
    par = cur;
    e_cur = at;
    cur = ce.y;
    pos += ce.w;
  }
  const int4 nd = s.node[cur];
  if (nd.w == 0) {
    s.n_absent += 1;
    return OP_DONE;
  }
  if (cur == 0 || nd.w > 1 || nd.y >= 2) {
    if (lane == 0) s.node[cur].w = nd.w - 1;
    __syncwarp();
    return OP_DONE;
  }
  if (nd.y == 1) {  // no sequence ends here any more and one child is left: fold the child in
    const int64_t need = adjacent_labels(s, e_cur, nd.x) ? 0 : (int64_t)s.child[e_cur].w + s.child[nd.x].w;
    if (!has_room(s, 0, 0, need)) return OP_NEED;
    merge_into_parent(s, cur, e_cur, lane);
    return OP_DONE;
  }
  // A leaf that stores nothing any more: unlink it from its parent.
  const int4 pn = s.node[par];
  const bool fold_parent = par != 0 && pn.w == 0 && pn.y == 2;
  if (fold_parent) {
    const int32_t other = (e_cur == pn.x) ? pn.x + 1 : pn.x;
    const int64_t need = adjacent_labels(s, e_par, other) ? 0 : (int64_t)s.child[e_par].w + s.child[other].w;
    if (!has_room(s, 0, 0, need)) return OP_NEED;
  }
  const int32_t leaf_label = s.child[e_cur].w;
  shift_down(s.child, (int64_t)e_cur + 1, (int64_t)pn.x + pn.y, lane);
  if (lane == 0) s.node[par].y = pn.y - 1;
  s.stale_child += nd.z;
  s.stale_label += leaf_label;
  free_node(s, cur, lane);
  __syncwarp();
  if (fold_parent) merge_into_parent(s, par, e_par, lane);
  return OP_DONE;
}

__global__ void __launch_bounds__(32) delta_kernel(TreeState* states, const int32_t* __restrict__ op,
                                                   const int64_t* __restrict__ seg_begin,
                                                   const int64_t* __restrict__ seg_off,
                                                   const int32_t* __restrict__ seg_len,
                                                   const int32_t* __restrict__ pool, int32_t* scratch,
                                                   int64_t stride) {
  const int lane = threadIdx.x;
  TreeState s = states[blockIdx.x];
  if (s.status != DELTA_OK || s.op_next >= s.op_end) return;
  int32_t* buf = scratch + (int64_t)blockIdx.x * stride;
  for (int64_t i = s.op_next; i < s.op_end; ++i) {
    int64_t n = 0;
    for (int64_t g = __ldg(seg_begin + i); g < __ldg(seg_begin + i + 1); ++g) {
      const int32_t* src = pool + __ldg(seg_off + g);
      const int32_t L = __ldg(seg_len + g);
      for (int32_t j = lane; j < L; j += 32) buf[n + j] = __ldg(src + j);
      n += L;
    }
    __syncwarp();
    const int r = __ldg(op + i) == 0 ? insert(s, buf, n, lane) : remove(s, buf, n, lane);
    if (r != OP_DONE) {
      s.status = r == OP_NEED ? DELTA_NEED_SPACE : DELTA_CORRUPT;
      s.op_next = i;
      break;
    }
    s.op_next = i + 1;
  }
  __syncwarp();
  if (lane == 0) states[blockIdx.x] = s;
}

__global__ void set_tree_kernel(TreeState* st, TreeView* view, TreeState v) {
  *st = v;
  *view = TreeView{v.node, v.child, v.label};
}

__global__ void refresh_views_kernel(const TreeState* st, TreeView* view, int32_t n) {
  const int32_t i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) view[i] = TreeView{st[i].node, st[i].child, st[i].label};
}

}  // namespace

cudaError_t launch_refresh_views(const TreeState* d_states, TreeView* d_views, int32_t n, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  refresh_views_kernel<<<(n + 127) / 128, 128, 0, st>>>(d_states, d_views, n);
  return cudaGetLastError();
}

cudaError_t launch_delta(TreeState* d_states, int32_t n_trees, const int32_t* op, const int64_t* seg_begin,
                         const int64_t* seg_off, const int32_t* seg_len, const int32_t* pool, int32_t* scratch,
                         int64_t scratch_stride, cudaStream_t st) {
  if (n_trees <= 0) return cudaSuccess;
  delta_kernel<<<n_trees, 32, 0, st>>>(d_states, op, seg_begin, seg_off, seg_len, pool, scratch, scratch_stride);
  return cudaGetLastError();
}

cudaError_t launch_set_tree(TreeState* d_state, TreeView* d_view, TreeState value, cudaStream_t st) {
  set_tree_kernel<<<1, 1, 0, st>>>(d_state, d_view, value);
  return cudaGetLastError();
}

}  // namespace p2p
