// lru_kernel.cu -- LRU eviction of a node's own cache trie on the device (EvictLRUTrie of Algorithm 1).
//
// Algorithm 1 evicts, while a request needs more memory than is free, the least recently used leaf token of
// the node's own trie, one token at a time (Section 2 primitive list: evictLRUTrie).  Every token's last
// access is the time of the latest insert (UpdateTrie) or served request (PrefixMatch) whose path covered it;
// ties go to the lexicographically smallest token path, and sequences that ended at an evicted token end one
// token earlier.
//
// Stamps.  A tree kept as an LRU cache has one stamp per node: the last access of every token of the node's
// edge.  An access that ends inside an edge splits it there (the upper part gets the new stamp; the node
// left between has one child and stores nothing -- the export merges such nodes back), so every edge's
// tokens share one stamp.  Times never decrease, so a token's stamp is never older than its descendants'.
//
// Eviction order without a token-by-token loop.  Let region(v) be the nodes of v's subtree reached from v
// through nodes of v's stamp, and end(v) the lexicographically largest token path in region(v) (follow the
// child with the largest first token among same-stamp children).  Removing the oldest leaf token n times
// removes the tokens in increasing order of (stamp, path of end, deeper first): a node becomes a leaf only
// after its descendants go, those of other stamps are older (removed before it) and those of its stamp
// include end(v), which precedes v in that order.  All tokens of one edge share the key, the deepest first.
// So n tokens are removed at once: the nodes whose key is below a threshold found by binary search on
// token counts, and the tail of the one node at the threshold.  The key's path order is the preorder rank
// of end(v) with children taken by first token.
//
// Kernels (all data-parallel; the host drives the level loops and the binary search):
//   lru_walk_kernel        warp per request: PrefixMatch, and per node the deepest touched position
//   lru_stamp_kernel       thread per node: stamp fully touched nodes, split partially touched edges
//   lru_bfs_kernel         warp per frontier node: children, parent links, child slots, next frontier
//   lru_size_kernel        subtree sizes, one level at a time from the deepest
//   lru_pairs/bitonic/runs/scan/off_kernel  sibling offsets: the (parent, first token) pairs sorted, sizes scanned
//   lru_rank_kernel        preorder ranks, one level at a time from the top
//   lru_end_kernel         end(v), one level at a time from the deepest
//   lru_count_kernel       token count of the nodes below a key (binary search steps)
//   lru_evict_kernel       one level at a time from the top: remove, cut the boundary edge, move terms
#include "internal.h"

namespace p2p {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kLruThreads = 256;
constexpr int32_t kTouchFull = INT32_MAX;

struct LruTree {
  int4* node;
  int4* child;
  const int32_t* label;
  const int32_t* shared;
  uint32_t* stamp;
};

__device__ __forceinline__ const int32_t* lab_of(const LruTree& t, int32_t off) {
  return label_ptr(t.label, t.shared, off);
}

// Live child with first token tok in the table at off (2^bits slots), one warp: 1 (entry, slot), 0 none.
__device__ int find_live(const LruTree& t, int32_t off, int32_t bits, int32_t tok, int lane, int4& e, int32_t& slot) {
  if (bits == 0) return 0;
  const uint32_t mask = (1u << bits) - 1, h = slot_hash(tok, bits);
  for (uint32_t base = 0; base <= mask; base += 32) {
    const uint32_t s = (h + base + lane) & mask;
    const int4 x = t.child[off + s];
    const unsigned hit = __ballot_sync(kFull, x.y >= 1 && x.x == tok);
    const unsigned empty = __ballot_sync(kFull, x.y == 0);
    const int fh = hit ? __ffs(hit) - 1 : 64, fe = empty ? __ffs(empty) - 1 : 64;
    if (fh < fe) {
      e.x = tok;
      e.y = __shfl_sync(kFull, x.y, fh);
      e.z = __shfl_sync(kFull, x.z, fh);
      e.w = __shfl_sync(kFull, x.w, fh);
      slot = off + (int32_t)((h + base + fh) & mask);
      return 1;
    }
    if (fe < 64) return 0;
  }
  return 0;
}

// First j in [0, lim) with a[j] != b[j], or lim (one warp).
__device__ int32_t first_mismatch(const int32_t* a, const int32_t* b, int32_t lim, int lane) {
  for (int32_t j0 = 0; j0 < lim; j0 += 32) {
    const int32_t j = j0 + lane;
    const unsigned m = __ballot_sync(kFull, j < lim && a[j] != b[j]);
    if (m) return j0 + __ffs(m) - 1;
  }
  return lim;
}

__global__ void __launch_bounds__(kLruThreads) lru_walk_kernel(LruTree t, const int32_t* __restrict__ tokens,
                                                               int64_t n_tokens, const int64_t* __restrict__ offsets,
                                                               int64_t B, int32_t* touch, int32_t* pslot,
                                                               int32_t* out_match, int32_t* err) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kLruThreads / 32);
  for (int64_t b = ((int64_t)blockIdx.x * kLruThreads + threadIdx.x) >> 5; b < B; b += warps) {
    const int64_t start = offsets[b], end = offsets[b + 1];
    if (!(start >= 0 && start <= end && end <= n_tokens && end - start <= INT32_MAX)) {
      if (lane == 0) {
        if (out_match) out_match[b] = 0;
        atomicOr(err, ERR_BAD_OFFSETS);
      }
      continue;
    }
    const int32_t* req = tokens + start;
    const int32_t len = (int32_t)(end - start);
    int4 nd = t.node[0];
    int32_t pos = 0;
    for (int guard = 0; pos < len && guard <= len; ++guard) {
      int4 e;
      int32_t slot;
      if (!find_live(t, nd.x, tab_bits(nd.y), req[pos], lane, e, slot)) break;
      const int32_t lim = min(e.w, len - pos);
      const int32_t k = first_mismatch(lab_of(t, e.z), req + pos, lim, lane);
      if (k == e.w) {
        if (lane == 0) atomicMax(&touch[e.y], kTouchFull);
        pos += k;
        nd = t.node[e.y];
        continue;
      }
      if (lane == 0 && k > 0) {  // the access ends inside this edge: its first k tokens are touched
        atomicMax(&touch[e.y], k);
        pslot[e.y] = slot;  // every toucher writes the same slot (the edge's own)
      }
      pos += k;
      break;
    }
    if (lane == 0 && out_match) out_match[b] = pos;
  }
}

// Thread per node v >= 1 (n_node: the node count before this call's splits).  Fully touched: stamp t.
// Partially touched at k: a new node mid takes the edge's first k tokens (stamp t) and has v, with the
// rest of the edge, as its one child.  Room for one node and one 4-slot table per split is ensured by the host.
__global__ void __launch_bounds__(kLruThreads) lru_stamp_kernel(LruTree t, TreeState* st, const int32_t* touch,
                                                                const int32_t* pslot, int32_t n_node, uint32_t time) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t v = 1 + (int64_t)blockIdx.x * kLruThreads + threadIdx.x; v < n_node; v += stride) {
    const int32_t k = touch[v];
    if (k == 0) continue;
    if (k == kTouchFull) {
      t.stamp[v] = time;
      continue;
    }
    const int32_t s = pslot[v];
    const int4 e = t.child[s];
    const int32_t mid = atomicAdd(&st->n_node, 1);
    const int32_t c0 = atomicAdd(&st->n_child, 1 << kMinTabBits);
    for (int j = 0; j < (1 << kMinTabBits); ++j) t.child[c0 + j] = make_int4(0, 0, 0, 0);
    const int4 lower = make_int4(lab_of(t, e.z)[k], (int32_t)v, label_adv(e.z, k), e.w - k);
    t.child[c0 + slot_hash(lower.x, kMinTabBits)] = lower;
    t.node[mid] = make_int4(c0, make_meta(kMinTabBits, 1), 1, 0);
    t.stamp[mid] = time;
    t.child[s] = make_int4(e.x, mid, e.z, k);
  }
}

// Warp per node of the frontier: its live children get parent and slot, and go to the next frontier (at most
// cap entries are written; the host checks the count against it).
__global__ void __launch_bounds__(kLruThreads) lru_bfs_kernel(LruTree t, const int32_t* __restrict__ front,
                                                              int32_t n_front, int32_t* next, int32_t* n_next,
                                                              int32_t cap, int32_t* parent, int32_t* cslot) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kLruThreads / 32);
  for (int64_t i = ((int64_t)blockIdx.x * kLruThreads + threadIdx.x) >> 5; i < n_front; i += warps) {
    const int32_t v = front[i];
    const int4 nd = t.node[v];
    const int32_t bits = tab_bits(nd.y);
    if (bits == 0) continue;
    for (int32_t b0 = 0; b0 < (1 << bits); b0 += 32) {
      const int32_t s = b0 + lane;
      const int4 x = s < (1 << bits) ? t.child[nd.x + s] : make_int4(0, 0, 0, 0);
      const bool live = x.y >= 1;
      const unsigned m = __ballot_sync(kFull, live);
      if (!m) continue;
      int32_t base = 0;
      if (lane == 0) base = atomicAdd(n_next, __popc(m));
      base = __shfl_sync(kFull, base, 0);
      const int32_t at = base + __popc(m & ((1u << lane) - 1));
      if (live && at < cap) {
        next[at] = x.y;
        parent[x.y] = v;
        cslot[x.y] = nd.x + s;
      }
    }
  }
}

// Nodes of one level add their subtree sizes to their parents (size starts at 1).
__global__ void __launch_bounds__(kLruThreads) lru_size_kernel(const int32_t* __restrict__ lvl, int32_t n,
                                                               const int32_t* __restrict__ parent, int64_t* size) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t i = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; i < n; i += stride) {
    const int32_t v = lvl[i];
    atomicAdd((unsigned long long*)&size[parent[v]], (unsigned long long)size[v]);
  }
}

// Sibling offsets for the preorder ranks: off[c] = the total subtree size of c's siblings whose first token
// is smaller (signed order).  All (parent, first token) pairs of the tree are sorted at once (a bitonic sort:
// a pair per live non-root node, padded to a power of two with the largest key), so each parent's children
// form one run in first-token order; off[c] is then an exclusive scan of the sizes in that order, less the
// scan at the start of c's run.  O(n log^2 n) for any fan-out.
__global__ void __launch_bounds__(kLruThreads) lru_pairs_kernel(LruTree t, const int32_t* __restrict__ nodes, int32_t n,
                                                                int64_t n2, const int32_t* __restrict__ parent,
                                                                const int32_t* __restrict__ cslot,
                                                                unsigned long long* key, int32_t* val) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t i = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; i < n2; i += stride) {
    if (i < n) {
      const int32_t v = nodes[i];
      const uint32_t tok = (uint32_t)t.child[cslot[v]].x ^ 0x80000000u;  // signed order as unsigned
      key[i] = ((unsigned long long)(uint32_t)parent[v] << 32) | tok;
      val[i] = v;
    } else {
      key[i] = ~0ull;
      val[i] = -1;
    }
  }
}

// One compare-exchange step of the bitonic sort of (key, val) over n2 (a power of two) entries.
__global__ void __launch_bounds__(kLruThreads) lru_bitonic_kernel(unsigned long long* key, int32_t* val, int64_t n2,
                                                                  int64_t j, int64_t k) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t i = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; i < n2; i += stride) {
    const int64_t l = i ^ j;
    if (l <= i) continue;
    const unsigned long long a = key[i], b = key[l];
    if ((a > b) == ((i & k) == 0)) {
      key[i] = b;
      key[l] = a;
      const int32_t va = val[i];
      val[i] = val[l];
      val[l] = va;
    }
  }
}

// For the sorted pairs [0, n): the first position of each parent's run (first[parent]) and the sizes in
// sorted order (into scan, scanned next).
__global__ void __launch_bounds__(kLruThreads) lru_runs_kernel(const unsigned long long* __restrict__ key,
                                                               const int32_t* __restrict__ val, int32_t n,
                                                               const int64_t* __restrict__ size, int32_t* first,
                                                               int64_t* scan) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t i = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; i < n; i += stride) {
    if (i == 0 || (key[i] >> 32) != (key[i - 1] >> 32)) first[(int32_t)(key[i] >> 32)] = (int32_t)i;
    scan[i] = size[val[i]];
  }
}

// Exclusive scan of scan[0, n) in place, one CTA: each thread sums a contiguous stretch, the CTA scans the
// stretch sums, each thread rewrites its stretch.
__global__ void __launch_bounds__(1024) lru_scan_kernel(int64_t* scan, int32_t n) {
  __shared__ int64_t s_part[1024];
  const int32_t per = (n + 1023) / 1024, a = min(n, (int32_t)threadIdx.x * per), b = min(n, a + per);
  int64_t sum = 0;
  for (int32_t i = a; i < b; ++i) sum += scan[i];
  s_part[threadIdx.x] = sum;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {  // inclusive scan of the stretch sums (Hillis-Steele)
    const int64_t x = threadIdx.x >= (unsigned)o ? s_part[threadIdx.x - o] : 0;
    __syncthreads();
    s_part[threadIdx.x] += x;
    __syncthreads();
  }
  int64_t run = s_part[threadIdx.x] - sum;
  for (int32_t i = a; i < b; ++i) {
    const int64_t x = scan[i];
    scan[i] = run;
    run += x;
  }
}

// off[c] for every sorted pair: the scan at c less the scan at the start of its parent's run.
__global__ void __launch_bounds__(kLruThreads) lru_off_kernel(const unsigned long long* __restrict__ key,
                                                              const int32_t* __restrict__ val, int32_t n,
                                                              const int32_t* __restrict__ first,
                                                              const int64_t* __restrict__ scan, int64_t* off) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t i = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; i < n; i += stride)
    off[val[i]] = scan[i] - scan[first[(int32_t)(key[i] >> 32)]];
}

// Preorder ranks of one level: rank[v] = rank[parent] + 1 + the sizes of v's earlier siblings.
__global__ void __launch_bounds__(kLruThreads) lru_rank_kernel(const int32_t* __restrict__ lvl, int32_t n,
                                                               const int32_t* __restrict__ parent,
                                                               const int64_t* __restrict__ off, int64_t* rank) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t i = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; i < n; i += stride) {
    const int32_t v = lvl[i];
    rank[v] = rank[parent[v]] + 1 + off[v];
  }
}

// end(v) for one level (its children's ends are final): the end of the same-stamp child with the largest
// first token, or v.  Then v offers itself to its parent when their stamps agree (best[] holds the offer
// with the largest first token: sign-flipped token in the high word, node in the low word).
__global__ void __launch_bounds__(kLruThreads) lru_end_kernel(LruTree t, const int32_t* __restrict__ lvl, int32_t n,
                                                              const int32_t* __restrict__ parent,
                                                              const int32_t* __restrict__ cslot,
                                                              unsigned long long* best, int32_t* end) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t i = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; i < n; i += stride) {
    const int32_t v = lvl[i];
    const unsigned long long bv = best[v];
    const int32_t e = bv ? end[(int32_t)(bv & 0xffffffffull)] : v;
    end[v] = e;
    const int32_t p = parent[v];
    if (p != 0 && t.stamp[v] == t.stamp[p]) {
      const uint32_t key = (uint32_t)t.child[cslot[v]].x ^ 0x80000000u;
      atomicMax(&best[p], ((unsigned long long)key << 32) | (uint32_t)v);
    }
  }
}

// The eviction key below stamp: (preorder rank of end(v), deeper first), one 64-bit word.
__device__ __forceinline__ unsigned long long key2_of(const int64_t* rank, const int32_t* end, int32_t v) {
  return ((unsigned long long)rank[end[v]] << 32) | (unsigned long long)(0xffffffffu - (uint32_t)rank[v]);
}

// Token count (edge lengths) of the non-root nodes nodes[0 .. n) with stamp < S (mode 0), or with stamp == S
// and key2 < K (mode 1), added to *out.
__global__ void __launch_bounds__(kLruThreads) lru_count_kernel(LruTree t, const int32_t* __restrict__ nodes, int32_t n,
                                                                const int32_t* __restrict__ cslot,
                                                                const int64_t* __restrict__ rank,
                                                                const int32_t* __restrict__ end, int mode, uint32_t S,
                                                                unsigned long long K, unsigned long long* out) {
  unsigned long long sum = 0;
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t i = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; i < n; i += stride) {
    const int32_t v = nodes[i];
    const uint32_t s = t.stamp[v];
    const bool in = mode == 0 ? s < S : (s == S && key2_of(rank, end, v) < K);
    if (in) sum += (unsigned long long)t.child[cslot[v]].w;
  }
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(kFull, sum, o);
  if ((threadIdx.x & 31) == 0 && sum) atomicAdd(out, sum);
}

// One level, from the top: a node below the threshold (stamp < S, or stamp == S and key2 < K) is removed --
// tombstoned in its parent's table when the parent stays -- and its stored sequences move to the nearest
// node that stays (surv); the node at the threshold (stamp == S, key2 == K) loses its last `cut` tokens.
__global__ void __launch_bounds__(kLruThreads) lru_evict_kernel(LruTree t, TreeState* st, const int32_t* __restrict__ lvl,
                                                                int32_t n, const int32_t* __restrict__ parent,
                                                                const int32_t* __restrict__ cslot,
                                                                const int64_t* __restrict__ rank,
                                                                const int32_t* __restrict__ end, uint32_t S,
                                                                unsigned long long K, int32_t cut, uint8_t* gone,
                                                                int32_t* surv) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t i = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; i < n; i += stride) {
    const int32_t v = lvl[i];
    const uint32_t s = t.stamp[v];
    const unsigned long long k2 = s == S ? key2_of(rank, end, v) : 0ull;
    const bool out = s < S || (s == S && k2 < K);
    gone[v] = out;
    if (!out) {
      if (s == S && k2 == K && cut > 0) t.child[cslot[v]].w -= cut;
      continue;
    }
    const int32_t p = parent[v];
    const int32_t sv = gone[p] ? surv[p] : p;
    surv[v] = sv;
    const int4 e = t.child[cslot[v]];
    if (!gone[p]) {
      t.child[cslot[v]].y = -1;  // tombstone: the slot keeps its key
      atomicSub(&t.node[p].z, 1);
    }
    const int4 nd = t.node[v];
    if (nd.w) atomicAdd(&t.node[sv].w, nd.w);
    atomicAdd((unsigned long long*)&st->dead_nodes, 1ull);
    if (e.z >= 0) atomicAdd((unsigned long long*)&st->stale_label, (unsigned long long)e.w);
    if (tab_bits(nd.y)) atomicAdd((unsigned long long*)&st->stale_child, 1ull << tab_bits(nd.y));
  }
}

// Node arrays of an eviction: size 1, the rest 0 (nodes of the BFS order).
__global__ void __launch_bounds__(kLruThreads) lru_init_kernel(const int32_t* __restrict__ order, int32_t n, int64_t* size,
                                                               int64_t* off, int64_t* rank, unsigned long long* best,
                                                               uint8_t* gone) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t i = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; i < n; i += stride) {
    const int32_t v = order[i];
    size[v] = 1;
    off[v] = 0;
    rank[v] = 0;
    best[v] = 0;
    gone[v] = 0;
  }
}

// A batch as INSERT ops of one tree: op i = request i, one pool run (its tokens); a request with invalid
// offsets gets a negative run length, which the delta validation rejects.
__global__ void __launch_bounds__(kLruThreads) lru_ops_kernel(const int64_t* __restrict__ offsets, int64_t B,
                                                              int64_t n_tokens, int32_t* op, int64_t* seg_begin,
                                                              int64_t* seg_off, int32_t* seg_len) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t b = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; b <= B; b += stride) {
    seg_begin[b] = b;
    if (b == B) continue;
    const int64_t s = offsets[b], e = offsets[b + 1];
    const bool ok = s >= 0 && s <= e && e <= n_tokens && e - s <= INT32_MAX;
    op[b] = P2P_OP_INSERT;
    seg_off[b] = ok ? s : 0;
    seg_len[b] = ok ? (int32_t)(e - s) : -1;
  }
}

// Section 5's expected hit rate of each routed request: the share of its tokens its target already holds,
// match[b][peer[b]] / |r_b| (IEEE single precision, rounded to nearest); 0 for an empty or unrouted request.
__global__ void __launch_bounds__(kLruThreads) hit_rate_kernel(const int32_t* __restrict__ match, int32_t P,
                                                               const int64_t* __restrict__ offsets, int64_t B,
                                                               const int32_t* __restrict__ peer, float* out) {
  const int64_t stride = (int64_t)gridDim.x * kLruThreads;
  for (int64_t b = (int64_t)blockIdx.x * kLruThreads + threadIdx.x; b < B; b += stride) {
    const int64_t len = offsets[b + 1] - offsets[b];
    const int32_t k = peer[b];
    out[b] = (k >= 0 && k < P && len > 0) ? __fdiv_rn((float)match[b * P + k], (float)len) : 0.0f;
  }
}

inline int grid_for(int64_t n, int per, int num_sms) {
  return (int)std::max<int64_t>(1, std::min<int64_t>((n + per - 1) / per, (int64_t)num_sms * 8));
}
inline LruTree lru_tree(const TreeState& s, const int32_t* shared) {
  return LruTree{s.node, s.child, s.label, shared, s.stamp};
}

}  // namespace

cudaError_t launch_lru_walk(const TreeState& s, const int32_t* shared, const int32_t* tokens, int64_t n_tokens,
                            const int64_t* offsets, int64_t B, int32_t* touch, int32_t* pslot, int32_t* out_match,
                            int32_t* err, int num_sms, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  P2P_TIMED(K_LRU_WALK, st,
            (lru_walk_kernel<<<grid_for(B, kLruThreads / 32, num_sms), kLruThreads, 0, st>>>(
                lru_tree(s, shared), tokens, n_tokens, offsets, B, touch, pslot, out_match, err)));
  return cudaGetLastError();
}

cudaError_t launch_lru_stamp(const TreeState& s, TreeState* d_state, const int32_t* shared, const int32_t* touch,
                             const int32_t* pslot, int32_t n_node, uint32_t time, int num_sms, cudaStream_t st) {
  if (n_node <= 1) return cudaSuccess;
  P2P_TIMED(K_LRU_STAMP, st,
            (lru_stamp_kernel<<<grid_for(n_node, kLruThreads, num_sms), kLruThreads, 0, st>>>(
                lru_tree(s, shared), d_state, touch, pslot, n_node, time)));
  return cudaGetLastError();
}

cudaError_t launch_lru_bfs(const TreeState& s, const int32_t* front, int32_t n_front, int32_t* next, int32_t* n_next,
                           int32_t cap, int32_t* parent, int32_t* cslot, int num_sms, cudaStream_t st) {
  if (n_front <= 0) return cudaSuccess;
  P2P_TIMED(K_LRU_ORDER, st,
            (lru_bfs_kernel<<<grid_for(n_front, kLruThreads / 32, num_sms), kLruThreads, 0, st>>>(
                lru_tree(s, nullptr), front, n_front, next, n_next, cap, parent, cslot)));
  return cudaGetLastError();
}

cudaError_t launch_lru_levels(const TreeState& s, const int32_t* order, const int32_t* lvl_begin, int32_t n_levels,
                              const int32_t* parent, const int32_t* cslot, int64_t* size, int64_t* off, int64_t* rank,
                              unsigned long long* best, int32_t* end, const LruSortScratch& sc, int num_sms,
                              cudaStream_t st) {
  const LruTree t = lru_tree(s, nullptr);
  // Sizes, from the deepest level up (level 0 is the root).
  for (int32_t l = n_levels - 1; l >= 1; --l) {
    const int32_t n = lvl_begin[l + 1] - lvl_begin[l];
    P2P_TIMED(K_LRU_ORDER, st,
              (lru_size_kernel<<<grid_for(n, kLruThreads, num_sms), kLruThreads, 0, st>>>(order + lvl_begin[l], n,
                                                                                          parent, size)));
  }
  // Sibling offsets (all parents at once, by a sort of the (parent, first token) pairs), then preorder ranks
  // from the top.
  const int32_t m = lvl_begin[n_levels] - 1;  // the live non-root nodes: order[1 .. m]
  if (m > 0) {
    int64_t n2 = 1;
    while (n2 < m) n2 <<= 1;
    P2P_TIMED(K_LRU_ORDER, st,
              (lru_pairs_kernel<<<grid_for(n2, kLruThreads, num_sms), kLruThreads, 0, st>>>(
                  t, order + 1, m, n2, parent, cslot, sc.key, sc.val)));
    for (int64_t k = 2; k <= n2; k <<= 1)
      for (int64_t j = k >> 1; j > 0; j >>= 1)
        P2P_TIMED(K_LRU_ORDER, st,
                  (lru_bitonic_kernel<<<grid_for(n2, kLruThreads, num_sms), kLruThreads, 0, st>>>(sc.key, sc.val, n2,
                                                                                                  j, k)));
    P2P_TIMED(K_LRU_ORDER, st,
              (lru_runs_kernel<<<grid_for(m, kLruThreads, num_sms), kLruThreads, 0, st>>>(sc.key, sc.val, m, size,
                                                                                         sc.first, sc.scan)));
    P2P_TIMED(K_LRU_ORDER, st, (lru_scan_kernel<<<1, 1024, 0, st>>>(sc.scan, m)));
    P2P_TIMED(K_LRU_ORDER, st,
              (lru_off_kernel<<<grid_for(m, kLruThreads, num_sms), kLruThreads, 0, st>>>(sc.key, sc.val, m, sc.first,
                                                                                        sc.scan, off)));
  }
  for (int32_t l = 1; l < n_levels; ++l) {
    const int32_t n = lvl_begin[l + 1] - lvl_begin[l];
    P2P_TIMED(K_LRU_ORDER, st,
              (lru_rank_kernel<<<grid_for(n, kLruThreads, num_sms), kLruThreads, 0, st>>>(order + lvl_begin[l], n,
                                                                                          parent, off, rank)));
  }
  // end(v), from the deepest level up.
  for (int32_t l = n_levels - 1; l >= 1; --l) {
    const int32_t n = lvl_begin[l + 1] - lvl_begin[l];
    P2P_TIMED(K_LRU_ORDER, st,
              (lru_end_kernel<<<grid_for(n, kLruThreads, num_sms), kLruThreads, 0, st>>>(t, order + lvl_begin[l], n,
                                                                                         parent, cslot, best, end)));
  }
  return cudaGetLastError();
}

cudaError_t launch_lru_count(const TreeState& s, const int32_t* nodes, int32_t n, const int32_t* cslot,
                             const int64_t* rank, const int32_t* end, int mode, uint32_t S, unsigned long long K,
                             unsigned long long* out, int num_sms, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(out, 0, sizeof(unsigned long long), st);
  if (e != cudaSuccess || n <= 0) return e;
  P2P_TIMED(K_LRU_SELECT, st,
            (lru_count_kernel<<<grid_for(n, kLruThreads, num_sms), kLruThreads, 0, st>>>(
                lru_tree(s, nullptr), nodes, n, cslot, rank, end, mode, S, K, out)));
  return cudaGetLastError();
}

cudaError_t launch_lru_evict(const TreeState& s, TreeState* d_state, const int32_t* order, const int32_t* lvl_begin,
                             int32_t n_levels, const int32_t* parent, const int32_t* cslot, const int64_t* rank,
                             const int32_t* end, uint32_t S, unsigned long long K, int32_t cut, uint8_t* gone,
                             int32_t* surv, int num_sms, cudaStream_t st) {
  for (int32_t l = 1; l < n_levels; ++l) {
    const int32_t n = lvl_begin[l + 1] - lvl_begin[l];
    P2P_TIMED(K_LRU_EVICT, st,
              (lru_evict_kernel<<<grid_for(n, kLruThreads, num_sms), kLruThreads, 0, st>>>(
                  lru_tree(s, nullptr), d_state, order + lvl_begin[l], n, parent, cslot, rank, end, S, K, cut, gone,
                  surv)));
  }
  return cudaGetLastError();
}

cudaError_t launch_lru_init(const int32_t* order, int32_t n, int64_t* size, int64_t* off, int64_t* rank,
                            unsigned long long* best, uint8_t* gone, int num_sms, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  P2P_TIMED(K_LRU_ORDER, st,
            (lru_init_kernel<<<grid_for(n, kLruThreads, num_sms), kLruThreads, 0, st>>>(order, n, size, off, rank, best,
                                                                                        gone)));
  return cudaGetLastError();
}

cudaError_t launch_lru_ops(const int64_t* offsets, int64_t B, int64_t n_tokens, int32_t* op, int64_t* seg_begin,
                           int64_t* seg_off, int32_t* seg_len, int num_sms, cudaStream_t st) {
  P2P_TIMED(K_LRU_OPS, st,
            (lru_ops_kernel<<<grid_for(B + 1, kLruThreads, num_sms), kLruThreads, 0, st>>>(offsets, B, n_tokens, op,
                                                                                           seg_begin, seg_off,
                                                                                           seg_len)));
  return cudaGetLastError();
}

cudaError_t launch_hit_rate(const int32_t* match, int32_t P, const int64_t* offsets, int64_t B, const int32_t* peer,
                            float* out, int num_sms, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  P2P_TIMED(K_HIT_RATE, st,
            (hit_rate_kernel<<<grid_for(B, kLruThreads, num_sms), kLruThreads, 0, st>>>(match, P, offsets, B, peer,
                                                                                        out)));
  return cudaGetLastError();
}

}  // namespace p2p
