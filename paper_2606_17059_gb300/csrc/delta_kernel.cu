// delta_kernel.cu -- anti-entropy delta applied to radix-tree replicas in HBM.
//
// An ordered list of ops patches one or more trees: INSERT adds one occurrence of a token sequence
// (updateTrie / updateTrieEstimate in the paper's Section 2 primitive list), DELETE removes one (a
// counted no-op when the sequence is not stored).  Trees stay edge-compressed and canonical: an INSERT
// that leaves an edge part-way splits it; a DELETE prunes a leaf that no longer stores anything and folds
// a node left with one child and no sequence into that child.
//
// Parallel schedule.  One CTA of kDeltaWarps warps takes a tree; the tree's ops are taken in chunks.
// Two facts make ops independent:
//   - ops on different sequences commute (the canonical tree depends only on the multiset), so only ops
//     on the same sequence must keep their order;
//   - two ops touch disjoint nodes when their paths part at some node and neither changes that node or
//     anything above it.
// Each chunk runs in two phases.
//   Parallel phase.  A read-only pre-walk finds, for every op, the first node with at least kWide
//   children on its path (its anchor, at most kAnchorDepth levels down).  Ops anchored at a node that
//   qualifies -- its table already fits the chunk's inserts under it (grown first if not) and it keeps at
//   least 3 children whatever the chunk's deletes under it do -- are bucketed by (anchor, next token) and
//   the warps take these sub-buckets concurrently.  They change only the anchor's table (slots claimed by
//   compare-and-swap, counters atomically) and the subtree of their own next token; nothing above the
//   anchor changes in this phase.  An op whose real walk does not pass through its anchor (the pre-walk
//   compares no labels) is deferred, untouched.
//   Serial phase.  The remaining ops, deferred ones included, are bucketed by a hash of their first token
//   (ops with different first tokens touch disjoint subtrees under the root and disjoint slots of the
//   root's table) and the warps take these buckets, heaviest first.
// Ops on the same sequence share an anchor and a next token, or a first token, so every bucket applies
// them in op order.  Inside an op the warp cooperates: a child lookup probes 32 table slots at once, labels
// are compared 256 tokens per step and copied 256 per step; lane 0 performs scalar stores and __syncwarp()
// orders them before later reads.  Adding or removing a child touches one slot (a table is doubled and
// rehashed when it passes 1/2 occupancy), so the cost of an op does not grow with the fan-out of the nodes
// it passes.
//
// Space.  Node, child-entry and label arenas are bump-allocated: each warp takes slabs from the tree's
// counters by compare-and-swap and hands out its ops' room from them; an op reserves everything it may
// need before it mutates anything.  If an arena is full the op
// is left undone, its bucket stops (as do, for the rest of the launch, the first-token buckets of every op
// it holds back, so no later op on the same sequence overtakes it) and the tree is flagged; the host grows
// the arenas and relaunches.  A per-op done flag records what is applied, so every op is applied whole,
// once.  Every loop is bounded by a sequence length, a list size or an iteration cap.
//
// Compaction (after the delta, when stale space passes live space): compact_kernel copies each tree's
// structure breadth-first into fresh arrays (one CTA per tree), then compact_labels_kernel moves the labels
// of all compacted trees over the whole GPU.
#include "internal.h"

namespace p2p {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kChunk = 3072;        // ops staged in shared memory at a time
constexpr int kWide = 4;            // children that make a node an anchor of parallel sub-buckets
constexpr int kAnchorDepth = 4;     // tree levels the pre-walk descends looking for an anchor
constexpr int kAnchorSlots = 768;  // distinct anchors per chunk (ops beyond stay in the serial phase)
constexpr int kSplitOps = 32;       // an anchor with this many ops in a chunk is split by next token
enum { OP_DONE = 0, OP_NEED = 1, OP_CORRUPT = 2, OP_DEFER = 3 };
enum { F_DONE = 1, F_ANCHORED = 2, F_DEFERRED = 4 };

// Tokens [0, na) come from a, [na, n) from b (an op's sequence as at most two pool runs).
struct Seq {
  const int32_t* a;
  const int32_t* b;
  int64_t na, n;
  bool pooled;  // a points into the delta's pool (not into gather scratch)
  __device__ int32_t at(int64_t i) const { return i < na ? a[i] : b[i - na]; }
};

// Per-warp view of one tree: array pointers and capacities (read-only during the kernel) and the
// tree's shared counters in global memory (updated atomically by the tree's warps).
struct Tree {
  int4* node;
  int4* child;
  int32_t* label;
  const int32_t* shared;  // router-wide pool of interned labels (read-only here)
  TreeState* g;
  int2* slab;  // this warp's slabs (shared memory): per counter, the next free unit and the units left
  __device__ const int32_t* lab(int32_t off) const { return label_ptr(label, shared, off); }
};

// Units a warp reserves at a time for its slab of counter c: nodes, child entries, label tokens.
__device__ __forceinline__ int32_t slab_units(int c) { return c == 0 ? 64 : c == 1 ? 256 : 4096; }

// Reserves k units of counter c (0 nodes, 1 child entries, 2 label tokens) from the tree's counters by
// compare-and-swap; -1 if they do not fit.  One lane.
__device__ int32_t reserve_units(const Tree& t, int c, int64_t k) {
  int32_t* ctr = c == 0 ? &t.g->n_node : c == 1 ? &t.g->n_child : &t.g->n_label;
  const int32_t cap = c == 0 ? t.g->cap_node : c == 1 ? t.g->cap_child : t.g->cap_label;
  int32_t old = *(volatile int32_t*)ctr;
  for (int it = 0; it < (1 << 20); ++it) {
    if ((int64_t)old + k > cap) return -1;
    const int32_t prev = atomicCAS(ctr, old, (int32_t)(old + k));
    if (prev == old) return old;
    old = prev;
  }
  return -1;
}

// Counts k units of counter c as stale (dead nodes, stale child entries, stale label tokens).  One lane.
__device__ void add_stale(const Tree& t, int c, int64_t k) {
  if (k <= 0) return;
  int64_t* p = c == 0 ? &t.g->dead_nodes : c == 1 ? &t.g->stale_child : &t.g->stale_label;
  atomicAdd((unsigned long long*)p, (unsigned long long)k);
}

// Reserves the room an op may need.  Each warp keeps a slab per counter, refilled slab_units(c) units at a
// time from the tree's counters (lanes 0, 1 and 2 at once), so most ops take their room without a global
// atomic; a slab's rest is counted as stale when it is replaced and when the warp finishes.  A request of a
// slab or more, or one whose refill does not fit, is reserved exactly.  On failure the op does nothing:
// room from a slab stays in it, room reserved exactly is counted as stale (a later compaction reclaims
// it), and the request is recorded for the host to grow the arenas.
__device__ bool take(Tree& t, int64_t nodes, int64_t entries, int64_t tokens, int32_t& n0, int32_t& c0, int32_t& l0,
                     int lane) {
  int32_t r = 0;
  int2 sl = make_int2(0, 0), ns = make_int2(0, 0);
  int64_t exact = 0;
  bool refilled = false;
  if (lane < 3) {
    const int64_t k = lane == 0 ? nodes : lane == 1 ? entries : tokens;
    sl = t.slab[lane];
    ns = sl;
    if (k > 0) {
      const int32_t S = slab_units(lane);
      if (k <= sl.y) {
        r = sl.x;
        ns = make_int2(sl.x + (int32_t)k, sl.y - (int32_t)k);
      } else if (k < S && (r = reserve_units(t, lane, S)) >= 0) {
        add_stale(t, lane, sl.y);
        refilled = true;
        ns = make_int2(r + (int32_t)k, S - (int32_t)k);
      } else {
        r = reserve_units(t, lane, k);
        exact = r >= 0 ? k : 0;
      }
    }
  }
  n0 = __shfl_sync(kFull, r, 0);
  c0 = __shfl_sync(kFull, r, 1);
  l0 = __shfl_sync(kFull, r, 2);
  const bool ok = n0 >= 0 && c0 >= 0 && l0 >= 0;
  if (lane < 3) {
    if (!ok) {
      if (exact) add_stale(t, lane, exact);
      ns = refilled ? make_int2(r, slab_units(lane)) : sl;
    }
    t.slab[lane] = ns;
  }
  __syncwarp();
  if (ok) return true;
  if (lane == 0) {
    atomicOr(&t.g->status, DELTA_NEED_SPACE);
    atomicMax(&t.g->need_node, (int32_t)nodes);
    atomicMax(&t.g->need_child, (int32_t)entries);
    atomicMax(&t.g->need_label, (int32_t)(tokens > INT32_MAX ? INT32_MAX : tokens));
  }
  return false;
}

// Looks `tok` up in the children table of 2^bits slots at child[off]: returns 1 (live child; e = its slot's
// entry), 2 (tombstone of tok), or 0 (absent; *slot = the first empty slot of its probe run, or -1 if there is
// none).  A slot is read as two 64-bit words (each single-copy atomic, the first holding key and state), so
// a slot another warp is claiming (root table only) is seen either all zero or with its final key.  Only
// this warp ever writes the slot of `tok` below this node, so the entry of a live `tok` is current.
__device__ int probe(const Tree& t, int32_t off, int32_t bits, int32_t tok, int lane, int32_t& slot, int4& e) {
  slot = -1;
  if (bits == 0) return 0;
  const uint32_t mask = (1u << bits) - 1, h = slot_hash(tok, bits);
  for (uint32_t base = 0; base <= mask; base += 32) {
    const uint32_t s = (h + base + lane) & mask;
    const longlong2 kv = __ldcv(reinterpret_cast<const longlong2*>(&t.child[off + s]));
    const int32_t key = (int32_t)(kv.x & 0xffffffffll), state = (int32_t)((unsigned long long)kv.x >> 32);
    const unsigned mine = __ballot_sync(kFull, key == tok && (state >= 1 || state == -1));
    const unsigned empty = __ballot_sync(kFull, state == 0);
    const int fm = mine ? __ffs(mine) - 1 : 64;
    const int fe = empty ? __ffs(empty) - 1 : 64;
    if (fm < fe) {
      slot = off + (int32_t)((h + base + fm) & mask);
      const long long a = __shfl_sync(kFull, kv.x, fm), b = __shfl_sync(kFull, kv.y, fm);
      e = make_int4((int32_t)(a & 0xffffffffll), (int32_t)((unsigned long long)a >> 32),
                    (int32_t)(b & 0xffffffffll), (int32_t)((unsigned long long)b >> 32));
      return e.y >= 1 ? 1 : 2;
    }
    if (fe < 64) {
      slot = off + (int32_t)((h + base + fe) & mask);
      return 0;
    }
  }
  return 0;
}

// Claims an empty slot for `tok` (64-bit compare-and-swap from all-zero, key written with the claim);
// re-probes if another warp took the slot first.  Returns the slot or -1.
__device__ int32_t claim(const Tree& t, int32_t off, int32_t bits, int32_t tok, int32_t slot, int lane) {
  const unsigned long long want = (unsigned long long)(uint32_t)tok | ((unsigned long long)(uint32_t)-3 << 32);
  for (int it = 0; it <= (1 << bits) && slot >= 0; ++it) {
    int32_t got = 0;
    if (lane == 0) got = atomicCAS((unsigned long long*)&t.child[slot], 0ull, want) == 0ull;
    if (__shfl_sync(kFull, got, 0)) return slot;
    int4 e;
    if (probe(t, off, bits, tok, lane, slot, e) != 0) return -1;
  }
  return -1;
}

// Publishes a claimed slot: label position first, then the child (the slot becomes live).
__device__ void publish(const Tree& t, int32_t slot, int32_t child_node, int32_t loff, int32_t llen, int lane) {
  if (lane == 0) {
    t.child[slot].z = loff;
    t.child[slot].w = llen;
    __threadfence();
    atomicExch(&t.child[slot].y, child_node);
  }
  __syncwarp();
}

// Writes the live entries of a table into a fresh all-zero table of 2^bits slots at child[dst] (lanes
// insert concurrently with compare-and-swap); returns false if an insertion found no slot.
__device__ bool rehash(const Tree& t, int32_t src, int32_t src_bits, int32_t dst, int32_t bits, int lane) {
  const uint32_t mask = (1u << bits) - 1;
  bool ok = true;
  for (int32_t j = lane; j < (1 << src_bits); j += 32) {
    const int4 e = t.child[src + j];
    if (e.y < 1) continue;
    const unsigned long long kv = (unsigned long long)(uint32_t)e.x | ((unsigned long long)(uint32_t)e.y << 32);
    uint32_t s = slot_hash(e.x, bits);
    bool placed = false;
    for (uint32_t it = 0; it <= mask && !placed; ++it, s = (s + 1) & mask) {
      if (atomicCAS((unsigned long long*)&t.child[dst + s], 0ull, kv) == 0ull) {
        t.child[dst + s].z = e.z;
        t.child[dst + s].w = e.w;
        placed = true;
      }
    }
    ok = ok && placed;
  }
  return __all_sync(kFull, ok);
}

__device__ void zero_slots(const Tree& t, int32_t off, int32_t n, int lane) {
  for (int32_t j = lane; j < n; j += 32) t.child[off + j] = make_int4(0, 0, 0, 0);
  __syncwarp();
}

// The single live child slot of a node's table (the node has exactly one child), skipping `except`.
__device__ int32_t only_child(const Tree& t, int32_t off, int32_t bits, int32_t except, int lane) {
  for (int32_t base = 0; base < (1 << bits); base += 32) {
    const int32_t j = base + lane;
    const bool live = j < (1 << bits) && off + j != except && t.child[off + j].y >= 1;
    const unsigned m = __ballot_sync(kFull, live);
    if (m) return off + base + __ffs(m) - 1;
  }
  return -1;
}

// Warp copies: 8 loads per lane in flight before their stores (256 tokens per step).
__device__ void copy_seq(int32_t* dst, const Seq& q, int64_t from, int64_t n, int lane) {
  for (int64_t j0 = 0; j0 < n; j0 += 256) {
    int32_t x[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int64_t j = j0 + u * 32 + lane;
      x[u] = j < n ? q.at(from + j) : 0;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int64_t j = j0 + u * 32 + lane;
      if (j < n) dst[j] = x[u];
    }
  }
}
__device__ void copy_tokens(int32_t* dst, const int32_t* src, int64_t n, int lane) {
  for (int64_t j0 = 0; j0 < n; j0 += 128) {
    int32_t x[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t j = j0 + u * 32 + lane;
      x[u] = j < n ? src[j] : 0;
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t j = j0 + u * 32 + lane;
      if (j < n) dst[j] = x[u];
    }
  }
}

// Label tokens are never overwritten once written (the label arena only grows) and the delta's pool is
// read-only, so "label[a .. a+n) == pool[b .. b+n)" stays true for the whole kernel once verified.  Each
// warp remembers the last such run; ops that walk the same shared prefix as the previous op (the common
// case: a delta references one pool copy of each shared prefix) skip re-comparing it.
constexpr int kMemoSlots = 16;  // verified runs each warp remembers

struct MemoEntry {
  const int32_t* lab;
  const int32_t* seq;
  int64_t n;
};
// A warp's memo: kMemoSlots entries in shared memory, so that the shared prefixes of the several anchors a
// warp serves all stay remembered.  Behind it, a table in global memory shared by every warp of the launch
// (all trees): runs verified from the start of an interned label (router-wide pool) against the start of a
// pool run of the delta.  The same prompt prefix is interned once for all replicas and sent once in the
// delta's pool, so it is compared once per launch instead of once per tree, chunk and anchor.  A key is
// (1 << 63 | pool offset of the label << 32 | pool offset of the run), claimed by compare-and-swap; its value
// only grows (atomicMax) and is always a verified length, so a reader that sees a key before its value
// reads 0 and merely compares.
constexpr int kGlobalMemoProbes = 8;
struct Memo {
  MemoEntry* e;
  unsigned long long* gkeys;  // NULL: no global table
  int32_t* gvals;
  uint32_t gmask;
  const int32_t* pool;
};

__device__ __forceinline__ unsigned long long global_memo_key(const Memo& m, const Seq& q, int32_t loff, int64_t pos) {
  if (!m.gkeys || loff >= 0 || !q.pooled) return 0ull;
  const int64_t soff = (q.a + pos) - m.pool;
  if (soff < 0 || soff > 0xffffffffll) return 0ull;
  return (1ull << 63) | ((unsigned long long)(uint32_t)~loff << 32) | (unsigned long long)soff;
}
__device__ __forceinline__ uint32_t global_memo_slot(unsigned long long key, uint32_t mask) {
  return (uint32_t)((key * 0x9E3779B97F4A7C15ull) >> 32) & mask;
}

// First j in [from, lim) with a[j] != b[j], or lim (one warp; both arrays contiguous in global memory).
// kDiffUnroll loads of 32 tokens in flight per lane and side; a block is folded into one OR of XORs per
// lane and one vote, and only a block that holds a mismatch is searched again.
constexpr int kDiffUnroll = 8;
__device__ int64_t first_diff_arrays(const int32_t* a, const int32_t* b, int64_t from, int64_t lim, int lane) {
  int64_t j0 = from;
  for (; j0 + 32 * kDiffUnroll <= lim; j0 += 32 * kDiffUnroll) {
    int32_t x[kDiffUnroll];
#pragma unroll
    for (int u = 0; u < kDiffUnroll; ++u) x[u] = a[j0 + u * 32 + lane];
    int32_t diff = 0;
#pragma unroll
    for (int u = 0; u < kDiffUnroll; ++u) diff |= x[u] ^ b[j0 + u * 32 + lane];
    if (__any_sync(kFull, diff != 0)) {
#pragma unroll
      for (int u = 0; u < kDiffUnroll; ++u) {
        const unsigned m = __ballot_sync(kFull, x[u] != b[j0 + u * 32 + lane]);
        if (m) return j0 + u * 32 + (__ffs(m) - 1);
      }
    }
  }
  for (; j0 < lim; j0 += 32) {
    const int64_t j = j0 + lane;
    const unsigned m = __ballot_sync(kFull, j < lim && a[j] != b[j]);
    if (m) return j0 + (__ffs(m) - 1);
  }
  return lim;
}

// First j in [from, lim) with lab[j] != q[pos + j], or lim.  Lane k looks at memo entry k, so a lookup is
// one step.  The sequence side is compared run by run (its first pool run, then the second), so both
// sides of every compare are contiguous.
__device__ int64_t first_diff(const int32_t* lab, int32_t loff, const Seq& q, int64_t pos, int64_t from, int64_t lim,
                              int lane, Memo& memo) {
  const bool in_a = pos < q.na;  // q[pos ..] starts in the first pool run, which the memo can describe
  const unsigned long long gkey = in_a ? global_memo_key(memo, q, loff, pos) : 0ull;
  if (in_a) {
    int32_t skip = 0;
    if (lane < kMemoSlots) {
      const MemoEntry m = memo.e[lane];
      const int64_t dl = lab - m.lab, ds = (q.a + pos) - m.seq;
      if (m.lab && dl == ds && dl >= 0 && dl < m.n) skip = (int32_t)min(lim, m.n - dl);
    }
    if (gkey && lane >= kMemoSlots && lane < kMemoSlots + kGlobalMemoProbes) {
      const uint32_t s = (global_memo_slot(gkey, memo.gmask) + (uint32_t)(lane - kMemoSlots)) & memo.gmask;
      if (__ldcg(memo.gkeys + s) == gkey) skip = (int32_t)min(lim, (int64_t)__ldcg(memo.gvals + s));
    }
    from = max(from, (int64_t)__reduce_max_sync(kFull, (unsigned)skip));
  }
  int64_t k = lim;
  if (from < lim) {
    const int64_t split = max(from, min(lim, q.na - pos));  // positions below split lie in the first run
    k = from < split ? first_diff_arrays(lab, q.a + pos, from, split, lane) : split;
    if (k == split && split < lim) k = first_diff_arrays(lab, q.b + (pos - q.na), split, lim, lane);
  }
  if (in_a && k >= 64) {  // remember a long verified run (within the first pool run), slot by label address
    if (lane == 0) {
      const int64_t nv = min(k, q.na - pos);
      const uint32_t h = (uint32_t)(((uintptr_t)lab >> 2) * 0x9E3779B97F4A7C15ull >> 32) & (kMemoSlots - 1);
      memo.e[h] = MemoEntry{lab, q.a + pos, nv};
      if (gkey) {
        const uint32_t h0 = global_memo_slot(gkey, memo.gmask);
        for (uint32_t i = 0; i < kGlobalMemoProbes; ++i) {
          const uint32_t s = (h0 + i) & memo.gmask;
          const unsigned long long prev = atomicCAS(memo.gkeys + s, 0ull, gkey);
          if (prev == 0ull || prev == gkey) {
            atomicMax(memo.gvals + s, (int32_t)min(nv, (int64_t)INT32_MAX));
            break;
          }
        }
      }
    }
    __syncwarp();
  }
  return k;
}

__device__ void add_stat(int64_t* p, int64_t v, int lane) {
  if (lane == 0 && v) atomicAdd((unsigned long long*)p, (unsigned long long)v);
}

// Labels a then b are one contiguous run (same label space, b starting where a ends): folding needs no copy.
__device__ bool adjacent(const int4& a, const int4& b) {
  if (a.z >= 0 && b.z >= 0) return (int64_t)a.z + a.w == b.z;
  if (a.z < 0 && b.z < 0) return (int64_t)~a.z + a.w == (int64_t)~b.z;
  return false;
}

// Node x (slot *ex in its parent's table) has one child and stores no sequence: fold the child's edge into
// x's.  The joined label is written at l0 unless the two labels are adjacent in the arena.
__device__ void fold_child(Tree& t, int32_t x, int4* ex, int32_t yslot, int32_t l0, int lane) {
  const int4 xe = *ex;
  const int4 xn = t.node[x];
  const int4 ye = t.child[yslot];
  const int4 yn = t.node[ye.y];
  int32_t off = xe.z;
  if (!adjacent(xe, ye)) {
    off = l0;
    copy_tokens(t.label + off, t.lab(xe.z), xe.w, lane);
    copy_tokens(t.label + off + xe.w, t.lab(ye.z), ye.w, lane);
    add_stat(&t.g->stale_label, (int64_t)xe.w + ye.w, lane);
  }
  __syncwarp();
  if (lane == 0) {
    ex->z = off;
    ex->w = xe.w + ye.w;
    t.node[x] = yn;
  }
  add_stat(&t.g->stale_child, tab_bits(xn.y) ? (int64_t)1 << tab_bits(xn.y) : 0, lane);
  add_stat(&t.g->dead_nodes, 1, lane);
  __syncwarp();
}

// Room for `extra` more children in node cur's table (cur != 0): grows the table (doubling, rehash into
// fresh slots) when claimed slots would pass 1/2, to at most 1/4 live load.  Returns false if the child
// arena is full.
__device__ bool ensure_room(Tree& t, int32_t cur, int4& nd, int32_t extra, int lane) {
  const int32_t bits = tab_bits(nd.y), used = tab_used(nd.y);
  if (!tab_full(bits, (int64_t)used + extra)) return true;
  int32_t nb = bits ? bits + 1 : kMinTabBits;
  while (nb < kMaxTabBits && ((int64_t)nd.z + extra) * 4 > ((int64_t)1 << nb)) ++nb;
  int32_t n0, c0, l0;
  if (!take(t, 0, (int64_t)1 << nb, 0, n0, c0, l0, lane)) return false;
  zero_slots(t, c0, 1 << nb, lane);
  if (bits && !rehash(t, nd.x, bits, c0, nb, lane)) return false;
  __syncwarp();
  add_stat(&t.g->stale_child, bits ? (int64_t)1 << bits : 0, lane);
  nd = make_int4(c0, make_meta(nb, nd.z), nd.z, nd.w);
  if (lane == 0) t.node[cur] = nd;
  __syncwarp();
  return true;
}

// A shortcut to an anchor, shared by the CTA's warps for one chunk's parallel phase.  Nothing above an
// anchor changes in that phase, so an op whose first pool run is the run (same address, same tokens) of
// the op that first reached the anchor, and covers the anchor's position, reaches it by the same path: it
// may start there.  The first op to reach the anchor claims the entry, writes pos and rec, and publishes
// seq last; the entry is not written again in the phase.
struct AnchorEntry {
  const int32_t* seq;  // the first pool run of the op that reached the anchor (NULL: not published)
  int32_t pos;         // tokens consumed on reaching it
  int32_t claim;
  int4 rec;            // its record then (its table offset and size hold for the phase)
};

// The shortcut test, taken by lane 0 for the whole warp: true (with pos and rec) if op q may start at the
// anchor of entry ae.
__device__ __forceinline__ bool anchor_start(const AnchorEntry* ae, const Seq& q, int lane, int64_t& pos, int4& rec) {
  int ok = 0;
  if (lane == 0 && ae) {
    const int32_t* sp = *(const int32_t* const volatile*)&ae->seq;
    ok = sp == q.a && sp != nullptr;
  }
  if (!__shfl_sync(kFull, ok, 0)) return false;
  __threadfence_block();
  pos = *(const volatile int32_t*)&ae->pos;
  rec = make_int4(*(const volatile int*)&ae->rec.x, *(const volatile int*)&ae->rec.y,
                  *(const volatile int*)&ae->rec.z, *(const volatile int*)&ae->rec.w);
  return q.na >= pos && q.n > pos;
}

// Publishes the shortcut for the op that first reached its anchor (at pos, record rec), if the entry is free
// and the op's first pool run covers the anchor's position.
__device__ __forceinline__ void anchor_publish(AnchorEntry* ae, const Seq& q, int64_t pos, const int4& rec, int lane) {
  if (lane == 0 && ae && pos <= q.na && atomicCAS(&ae->claim, 0, 1) == 0) {
    ae->pos = (int32_t)pos;
    ae->rec = rec;
    __threadfence_block();
    *(const int32_t* volatile*)&ae->seq = q.a;
  }
  __syncwarp();
}

// root: the root's node record as of the launch (its table moves only between launches).  anchor: in the
// parallel phase, the op's anchor node (else -1): the op changes nothing until its walk has passed through
// the anchor (OP_DEFER otherwise), and claims in the anchor's table are counted atomically.
__device__ int insert(Tree& t, const Seq& q, const int4& root, int32_t anchor, int lane, Memo& memo,
                      AnchorEntry* ae) {
  const int64_t n = q.n;
  if (n == 0) {
    if (lane == 0) atomicAdd(&t.node[0].w, 1);
    __syncwarp();
    return OP_DONE;
  }
  int32_t cur = 0;
  int64_t pos = 0;
  int32_t n0, c0, l0;
  int4 nd = root;  // record of node cur: below the root (and the anchor) only this warp writes it
  bool passed = anchor < 0;
  if (anchor >= 0 && anchor_start(ae, q, lane, pos, nd)) {
    cur = anchor;
    passed = true;
  } else {
    pos = 0;
    nd = root;
  }
  for (int64_t guard = 0; guard <= n + 1; ++guard) {
    if (pos == n) {  // the sequence ends exactly at node cur (never the root here: n > 0)
      if (!passed || cur == anchor) return OP_DEFER;
      if (lane == 0) t.node[cur].w += 1;
      __syncwarp();
      return OP_DONE;
    }
    const int32_t tok = q.at(pos);
    int32_t slot;
    int4 ce;
    int st = probe(t, nd.x, tab_bits(nd.y), tok, lane, slot, ce);
    if (st != 1) {
      // New leaf edge q[pos, n) under cur: revive tok's tombstone, or claim an empty slot.
      if (!passed) return OP_DEFER;
      const int64_t L = n - pos;
      if (st == 0) {
        if (cur == anchor) {
          // The anchor's table is shared by the parallel phase's warps and was sized for the chunk's
          // inserts under it: count the claim atomically; a table that would pass 1/2 defers the op.
          int32_t meta = 0;
          if (lane == 0) meta = atomicAdd(&t.node[cur].y, 1 << 5);
          meta = __shfl_sync(kFull, meta, 0);
          if (slot < 0 || tab_full(tab_bits(meta), (int64_t)tab_used(meta) + 1)) {
            if (lane == 0) atomicSub(&t.node[cur].y, 1 << 5);
            return OP_DEFER;
          }
        } else if (cur == 0) {
          // The root table is shared by all warps of the tree: count the claim atomically; if the table
          // would pass 1/2 the host grows it between launches.
          int32_t meta = 0;
          if (lane == 0) meta = atomicAdd(&t.node[0].y, 1 << 5);
          meta = __shfl_sync(kFull, meta, 0);
          if (slot < 0 || tab_full(tab_bits(meta), (int64_t)tab_used(meta) + 1)) {
            if (lane == 0) {
              atomicSub(&t.node[0].y, 1 << 5);
              atomicMax(&t.g->need_root, 1);
              atomicOr(&t.g->status, DELTA_NEED_SPACE);
            }
            return OP_NEED;
          }
        } else {
          if (!ensure_room(t, cur, nd, 1, lane)) return OP_NEED;
          st = probe(t, nd.x, tab_bits(nd.y), tok, lane, slot, ce);
          if (st != 0 || slot < 0) return OP_CORRUPT;
          if (lane == 0) t.node[cur].y = nd.y + (1 << 5);
        }
      }
      if (!take(t, 1, 0, L, n0, c0, l0, lane)) {
        if (st == 0 && lane == 0) atomicSub(&t.node[cur].y, 1 << 5);
        return OP_NEED;
      }
      copy_seq(t.label + l0, q, pos, L, lane);
      if (lane == 0) t.node[n0] = make_int4(0, 0, 0, 1);
      __syncwarp();
      if (st == 0 && (slot = claim(t, nd.x, tab_bits(nd.y), tok, slot, lane)) < 0) return OP_CORRUPT;
      if (cur == 0 && lane == 0) {  // a new first token at the root: the route kernels' filter must know it
        const uint32_t h = root_filter_bit(tok);
        atomicOr(t.g->rfilter + (h >> 5), 1u << (h & 31));
      }
      publish(t, slot, n0, l0, (int32_t)L, lane);
      if (lane == 0) atomicAdd(&t.node[cur].z, 1);
      __syncwarp();
      return OP_DONE;
    }
    int4* ent = t.child + slot;
    if (ce.w <= 0 || ce.y <= 0) return OP_CORRUPT;
    const int4 nn = t.node[ce.y];  // the child's record, fetched while the label is compared
    const int64_t lim = min((int64_t)ce.w, n - pos);
    const int64_t k = first_diff(t.lab(ce.z), ce.z, q, pos, 1, lim, lane, memo);
    if (k == ce.w) {
      cur = ce.y;
      pos += k;
      nd = nn;
      if (!passed && cur == anchor) {
        passed = true;
        anchor_publish(ae, q, pos, nd, lane);
      }
      continue;
    }
    // The sequence leaves (or ends inside) the edge after k tokens: split it there.  The new node mid
    // gets a 4-slot table holding the lower part of the edge (and the new leaf).
    if (!passed) return OP_DEFER;
    const bool tail = pos + k < n;
    const int64_t L = n - pos - k;
    if (!take(t, tail ? 2 : 1, 1 << kMinTabBits, tail ? L : 0, n0, c0, l0, lane)) return OP_NEED;
    const int32_t mid = n0, leaf = n0 + 1;
    zero_slots(t, c0, 1 << kMinTabBits, lane);
    const int4 lower = make_int4(t.lab(ce.z)[k], ce.y, label_adv(ce.z, (int32_t)k), ce.w - (int32_t)k);
    if (tail) copy_seq(t.label + l0, q, pos + k, L, lane);
    const int32_t leaf_tok = tail ? q.at(pos + k) : 0;
    __syncwarp();
    if (lane == 0) {
      const uint32_t mask = (1u << kMinTabBits) - 1;
      uint32_t s0 = slot_hash(lower.x, kMinTabBits);
      t.child[c0 + s0] = lower;
      if (tail) {
        uint32_t s1 = slot_hash(leaf_tok, kMinTabBits);
        while (s1 == s0) s1 = (s1 + 1) & mask;
        t.child[c0 + s1] = make_int4(leaf_tok, leaf, l0, (int32_t)L);
        t.node[leaf] = make_int4(0, 0, 0, 1);
      }
      t.node[mid] = make_int4(c0, make_meta(kMinTabBits, tail ? 2 : 1), tail ? 2 : 1, tail ? 0 : 1);
      __threadfence_block();
      ent->w = (int32_t)k;  // the slot keeps its key; label_off is unchanged
      atomicExch(&ent->y, mid);
    }
    __syncwarp();
    return OP_DONE;
  }
  return OP_CORRUPT;
}

// anchor as for insert: nothing changes (OP_DEFER) unless the walk passed through it, and the anchor is
// never folded here.
__device__ int remove(Tree& t, const Seq& q, const int4& root, int32_t anchor, int lane, Memo& memo,
                      AnchorEntry* ae) {
  const int64_t n = q.n;
  if (n == 0) {
    int ok = 0;
    if (lane == 0) {
      const int32_t old = atomicAdd(&t.node[0].w, -1);
      ok = old > 0;
      if (!ok) atomicAdd(&t.node[0].w, 1);
    }
    if (!__shfl_sync(kFull, ok, 0)) add_stat(&t.g->n_absent, 1, lane);
    __syncwarp();
    return OP_DONE;
  }
  int32_t cur = 0, par = -1, gpar = -1, s_gpar = -1;  // s_gpar: gpar's slot in its parent's table
  int4 *e_cur = nullptr, *e_par = nullptr;
  int64_t pos = 0;
  int4 nd = root, pn = root;  // records of cur and par (below the root and the anchor only this warp writes them)
  bool passed = anchor < 0;
  if (anchor >= 0 && anchor_start(ae, q, lane, pos, nd)) {
    cur = anchor;  // par and e_cur stay unknown: the anchor is never folded here
    passed = true;
  } else {
    pos = 0;
    nd = root;
  }
  for (int64_t guard = 0; pos < n; ++guard) {
    if (guard > n) return OP_CORRUPT;
    int32_t slot;
    int4 ce;
    if (probe(t, nd.x, tab_bits(nd.y), q.at(pos), lane, slot, ce) != 1) {
      if (!passed) return OP_DEFER;
      add_stat(&t.g->n_absent, 1, lane);
      return OP_DONE;
    }
    int4* ent = t.child + slot;
    if (ce.w <= 0 || ce.y <= 0) return OP_CORRUPT;
    const int4 nn = t.node[ce.y];  // the child's record, fetched while the label is compared
    if (pos + ce.w > n || first_diff(t.lab(ce.z), ce.z, q, pos, 1, ce.w, lane, memo) < ce.w) {
      if (!passed) return OP_DEFER;
      add_stat(&t.g->n_absent, 1, lane);
      return OP_DONE;
    }
    s_gpar = e_par ? (int32_t)(e_par - t.child) : -1;
    e_par = e_cur;
    gpar = par;
    par = cur;
    pn = nd;
    e_cur = ent;
    cur = ce.y;
    pos += ce.w;
    nd = nn;
    if (!passed && cur == anchor) {
      passed = true;
      anchor_publish(ae, q, pos, nd, lane);
    }
  }
  if (!passed || cur == anchor) return OP_DEFER;
  if (nd.w == 0) {
    add_stat(&t.g->n_absent, 1, lane);
    return OP_DONE;
  }
  if (nd.w > 1 || nd.z >= 2) {
    if (lane == 0) t.node[cur].w = nd.w - 1;
    __syncwarp();
    return OP_DONE;
  }
  int32_t n0, c0, l0;
  if (nd.z == 1) {  // no sequence ends here any more and one child is left: fold the child in
    const int32_t ys = only_child(t, nd.x, tab_bits(nd.y), -1, lane);
    if (ys < 0) return OP_CORRUPT;
    const int4 ce = *e_cur, ye = t.child[ys];
    const int64_t need = adjacent(ce, ye) ? 0 : (int64_t)ce.w + ye.w;
    if (!take(t, 0, 0, need, n0, c0, l0, lane)) return OP_NEED;
    fold_child(t, cur, e_cur, ys, l0, lane);
    return OP_DONE;
  }
  // A leaf that stores nothing any more: tombstone its slot in the parent's table.  (pn is only read when
  // par is not the root.)  A parent that stores nothing and has this leaf as its only child (a node an upload
  // put in front of a label's own rest, or an LRU access's split) would be left empty: it goes too, from its
  // own parent's table.
  // The parent goes too when it would be left empty: it stores nothing and this leaf is its only child (an
  // upload's node in front of a label's own rest).  Its own parent gpar then loses a child, and like any node
  // left with one child and no sequence it takes that child in (so no chain of such nodes ever forms, and a
  // removal never has to climb more than this one level).
  const bool drop_parent = par != 0 && pn.w == 0 && pn.z == 1;
  if (drop_parent && (gpar < 0 || !e_par)) return anchor >= 0 ? OP_DEFER : OP_CORRUPT;  // (cannot happen)
  const bool fold_parent = par != 0 && pn.w == 0 && pn.z == 2;
  if (fold_parent && par == anchor) return OP_DEFER;  // (cannot happen: an anchor keeps >= 3 children)
  int32_t other = -1;
  if (fold_parent) {
    other = only_child(t, pn.x, tab_bits(pn.y), (int32_t)(e_cur - t.child), lane);
    if (other < 0) return OP_CORRUPT;
    const int4 oe = t.child[other];
    const int64_t need = adjacent(*e_par, oe) ? 0 : (int64_t)e_par->w + oe.w;
    if (!take(t, 0, 0, need, n0, c0, l0, lane)) return OP_NEED;
  }
  // gpar below the anchor (or in the serial phase) is this warp's alone; an anchor keeps >= 3 children.
  int4 gpn = make_int4(0, 0, 0, 0);
  if (drop_parent && gpar != 0 && gpar != anchor) gpn = t.node[gpar];
  const bool fold_gpar = drop_parent && gpar != 0 && gpar != anchor && gpn.w == 0 && gpn.z == 2;
  if (fold_gpar) {
    if (s_gpar < 0) return anchor >= 0 ? OP_DEFER : OP_CORRUPT;  // (cannot happen: gpar was reached by a slot)
    other = only_child(t, gpn.x, tab_bits(gpn.y), (int32_t)(e_par - t.child), lane);
    if (other < 0) return OP_CORRUPT;
    const int4 oe = t.child[other], ge = t.child[s_gpar];
    const int64_t need = adjacent(ge, oe) ? 0 : (int64_t)ge.w + oe.w;
    if (!take(t, 0, 0, need, n0, c0, l0, lane)) return OP_NEED;
  }
  const int32_t leaf_label = e_cur->w;
  if (lane == 0) {
    atomicExch(&e_cur->y, -1);  // the slot keeps its key
    atomicAdd(&t.node[par].z, -1);
  }
  add_stat(&t.g->stale_label, leaf_label, lane);
  add_stat(&t.g->dead_nodes, 1, lane);
  add_stat(&t.g->stale_child, tab_bits(nd.y) ? (int64_t)1 << tab_bits(nd.y) : 0, lane);
  if (drop_parent) {
    if (lane == 0) {
      atomicExch(&e_par->y, -1);
      atomicAdd(&t.node[gpar].z, -1);
    }
    add_stat(&t.g->dead_nodes, 1, lane);
    add_stat(&t.g->stale_child, tab_bits(pn.y) ? (int64_t)1 << tab_bits(pn.y) : 0, lane);
  }
  __syncwarp();
  if (fold_parent) fold_child(t, par, e_par, other, l0, lane);
  if (fold_gpar) fold_child(t, gpar, t.child + s_gpar, other, l0, lane);
  return OP_DONE;
}

// Bucket of an op in the serial phase: a hash of the sequence's first token.
__device__ __forceinline__ int32_t bucket_of(int32_t tok) {
  return (int32_t)(((uint32_t)tok * 0x85EBCA6Bu) >> (32 - kDeltaBucketBits));
}
// Sub-bucket of an anchored op in the parallel phase: a hash of (anchor, next token) for an anchor with
// many ops in the chunk, else of the anchor alone (one warp then serves all of that anchor's ops, and its
// memo keeps their shared prefix).
__device__ __forceinline__ int32_t sub_bucket_of(int32_t anchor, int32_t tok, bool split) {
  const uint32_t h = ((uint32_t)anchor * 0x9E3779B1u) ^ (split ? (uint32_t)tok * 0x85EBCA6Bu : 0u);
  return (int32_t)((h * 0xC2B2AE35u) >> (32 - kDeltaBucketBits));
}

// Token pos of an op's sequence given by pool runs [g0, g1) (one thread); -1 past the end.
__device__ int32_t run_token(const int64_t* __restrict__ seg_off, const int32_t* __restrict__ seg_len,
                             const int32_t* __restrict__ pool, int64_t g0, int64_t g1, int64_t pos) {
  for (int64_t g = g0; g < g1; ++g) {
    const int32_t l = seg_len[g];
    if (pos < l) return pool[seg_off[g] + pos];
    pos -= l;
  }
  return -1;
}

// Read-only pre-walk of one op (one thread, no label compares): the first node with at least kWide
// children on the path that the sequence's tokens select, within kAnchorDepth levels, provided the sequence
// continues past it; anchor = -1 if there is none.  next_tok is the sequence's token just past the anchor.
__device__ void find_anchor(const Tree& t, const int4& root, const int64_t* __restrict__ seg_off,
                            const int32_t* __restrict__ seg_len, const int32_t* __restrict__ pool, int64_t g0,
                            int64_t g1, int64_t n, int32_t& anchor, int32_t& next_tok) {
  anchor = -1;
  next_tok = 0;
  int4 nd = root;
  int64_t pos = 0;
  for (int depth = 0; depth < kAnchorDepth && pos < n; ++depth) {
    const int32_t bits = tab_bits(nd.y);
    if (bits == 0) return;
    const int32_t tok = run_token(seg_off, seg_len, pool, g0, g1, pos);
    const uint32_t mask = (1u << bits) - 1;
    uint32_t sl = slot_hash(tok, bits);
    int4 ce = make_int4(0, 0, 0, 0);
    for (uint32_t it = 0; it <= mask; ++it, sl = (sl + 1) & mask) {
      const int4 e = __ldcg(t.child + nd.x + sl);
      if (e.y == 0) return;
      if (e.y >= 1 && e.x == tok) {
        ce = e;
        break;
      }
    }
    if (ce.y < 1 || ce.w <= 0) return;
    pos += ce.w;
    if (pos >= n) return;
    const int4 cn = __ldcg(t.node + ce.y);
    if (cn.z >= kWide) {
      anchor = ce.y;
      next_tok = run_token(seg_off, seg_len, pool, g0, g1, pos);
      return;
    }
    nd = cn;
  }
}

// Applies op i (one warp); anchor as for insert/remove.
__device__ int apply_op(Tree& t, const int4& root, int32_t anchor, int32_t opcode, int64_t g0, int64_t g1,
                        const int64_t* __restrict__ seg_off, const int32_t* __restrict__ seg_len,
                        const int32_t* __restrict__ pool, int32_t* buf, int lane, Memo& memo, AnchorEntry* ae) {
  // The op's sequence: up to two pool runs are read in place, more are gathered into scratch.
  Seq q;
  q.pooled = g1 - g0 <= 2;
  if (g1 - g0 <= 2) {
    q.a = pool + (g1 > g0 ? seg_off[g0] : 0);
    q.na = g1 > g0 ? seg_len[g0] : 0;
    q.b = g1 - g0 == 2 ? pool + seg_off[g0 + 1] : q.a;
    q.n = q.na + (g1 - g0 == 2 ? seg_len[g0 + 1] : 0);
  } else {
    if (!buf) return OP_CORRUPT;  // the host gives gather scratch whenever an op has more than two runs
    int64_t len = 0;
    for (int64_t g = g0; g < g1; ++g) {
      copy_tokens(buf + len, pool + seg_off[g], seg_len[g], lane);
      len += seg_len[g];
    }
    __syncwarp();
    q.a = q.b = buf;
    q.na = q.n = len;
  }
  return opcode == P2P_OP_INSERT ? insert(t, q, root, anchor, lane, memo, ae)
                                 : remove(t, q, root, anchor, lane, memo, ae);
}

// Lane 0 asks L1 for the op code and pool-run descriptors of the warp's next op (op jn of the chunk at c0)
// while the current op runs: the next op's first loads then hit in L1.  Only ops with a pool run are
// prefetched (their descriptor index is inside the arrays).
__device__ __forceinline__ void prefetch_op(const int32_t* op, const int64_t* seg_off, const int32_t* seg_len,
                                            const int64_t* s_run, int64_t c0, int jn, int lane) {
  if (lane != 0) return;
  const int64_t g0 = s_run[jn];
  asm volatile("prefetch.global.L1 [%0];" :: "l"(op + c0 + jn));
  if (s_run[jn + 1] > g0) {
    asm volatile("prefetch.global.L1 [%0];" :: "l"(seg_off + g0));
    asm volatile("prefetch.global.L1 [%0];" :: "l"(seg_len + g0));
  }
}

// Ranks kDeltaBuckets buckets by count (heaviest first, ties to the lower bucket) into order; one warp.
__device__ void rank_buckets(const int* count, int* order, int lane) {
  const int mine = count[lane];
  int rank = 0;
  for (int o = 0; o < kDeltaBuckets; ++o) {
    const int other = count[o];
    rank += other > mine || (other == mine && o < lane);
  }
  order[rank] = lane;
}

// Bytes of the delta kernel's dynamic shared memory (the chunk's per-op and per-anchor arrays).
constexpr int delta_smem_bytes() {
  return kAnchorSlots * (int)sizeof(AnchorEntry) + (kChunk + 1) * 8 + kChunk * 4 * 2 + kAnchorSlots * 4 * 4 +
         kChunk * 2 + kChunk * 1 * 2;
}

// kParts: the launch splits heavy trees among CTAs (parts); a separate instantiation, so that the ordinary
// launch keeps the code it had without the split.
template <bool kParts>
__global__ void __launch_bounds__(kDeltaWarps * 32, 2)
    delta_kernel(TreeState* states, uint8_t* done, const int32_t* __restrict__ op,
                 const int64_t* __restrict__ seg_begin, const int64_t* __restrict__ seg_off,
                 const int32_t* __restrict__ seg_len, const int32_t* __restrict__ pool, int32_t* gather,
                 int64_t stride, const int32_t* shared, unsigned long long* gmemo_keys, int32_t* gmemo_vals,
                 uint32_t gmemo_mask, const int32_t* __restrict__ parts) {
  // The chunk's per-op and per-anchor arrays, in dynamic shared memory (delta_smem_bytes()).
  extern __shared__ __align__(16) unsigned char s_dyn[];
  AnchorEntry* s_aentry = reinterpret_cast<AnchorEntry*>(s_dyn);        // per anchor: its shortcut
  int64_t* s_run = reinterpret_cast<int64_t*>(s_aentry + kAnchorSlots);  // seg_begin of the chunk's ops (+1)
  int32_t* s_anchor = reinterpret_cast<int32_t*>(s_run + kChunk + 1);    // anchor of an anchored op
  int32_t* s_next = s_anchor + kChunk;   // an anchored op's token just past its anchor, then its sub-bucket
  int* s_akey = s_next + kChunk;         // per anchor slot: the anchor, its inserts, deletes, qualification
  int* s_ains = s_akey + kAnchorSlots;
  int* s_adel = s_ains + kAnchorSlots;
  int* s_aok = s_adel + kAnchorSlots;
  int16_t* s_aslot = reinterpret_cast<int16_t*>(s_aok + kAnchorSlots);  // an op's entry in the anchor table
  int8_t* s_bucket = reinterpret_cast<int8_t*>(s_aslot + kChunk);       // first-token bucket
  uint8_t* s_flag = reinterpret_cast<uint8_t*>(s_bucket + kChunk);      // F_* bits
  __shared__ int s_count[kDeltaBuckets];
  __shared__ int s_order[kDeltaBuckets];
  __shared__ int s_stop[kDeltaBuckets];  // first-token buckets held back for the rest of the launch
  __shared__ int s_take;
  __shared__ int s_any;
  __shared__ MemoEntry s_memo[kDeltaWarps][kMemoSlots];
  __shared__ int2 s_slab[kDeltaWarps][3];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane < 3) s_slab[warp][lane] = make_int2(0, 0);
  // This CTA's tree, and its part of the tree's ops: the ops whose first-token bucket is `part` modulo
  // `nparts` (kDeltaBuckets buckets).  Ops with different first tokens touch disjoint subtrees and, of the
  // root, only its table, whose claims and counts are atomic; so the CTAs of one tree never touch the same
  // node below the root, and all ops on one sequence stay in one CTA, in op order.
  const int32_t pw = kParts ? parts[blockIdx.x] : (int32_t)blockIdx.x;
  const int32_t part = kParts ? (pw >> kPartShift) & 31 : 0, nparts = kParts ? (pw >> kNpartShift) & 63 : 1;
  TreeState* gs = states + (kParts ? (pw & kPartTreeMask) : pw);
  if (lane < kMemoSlots) s_memo[warp][lane] = MemoEntry{nullptr, nullptr, 0};
  const int64_t op_begin = gs->op_begin, op_end = gs->op_end;
  if (threadIdx.x == 0) s_any = 0;
  if (threadIdx.x < kDeltaBuckets) s_stop[threadIdx.x] = 0;
  __syncthreads();
  for (int64_t i = op_begin + threadIdx.x; i < op_end; i += blockDim.x)
    if (!done[i]) {
      s_any = 1;
      break;
    }
  __syncthreads();
  if (!s_any || gs->status & DELTA_CORRUPT) return;
  Tree t;
  t.node = gs->node;
  t.child = gs->child;
  t.label = gs->label;
  t.shared = shared;
  t.g = gs;
  t.slab = s_slab[warp];
  const int4 root = t.node[0];  // its table offset and size hold for the whole launch
  int32_t* buf = gather ? gather + ((int64_t)blockIdx.x * kDeltaWarps + warp) * stride : nullptr;
  // Facts about immutable labels: valid whichever bucket the warp works on.
  Memo memo{s_memo[warp], gmemo_keys, gmemo_vals, gmemo_mask, pool};
  for (int64_t c0 = op_begin; c0 < op_end; c0 += kChunk) {
    const int clen = (int)min((int64_t)kChunk, op_end - c0);
    // 1. Per op: first-token bucket, done flag, and (for ops still to apply) the anchor.
    for (int k = threadIdx.x; k < kAnchorSlots; k += blockDim.x) {
      s_akey[k] = -1;
      s_ains[k] = 0;
      s_adel[k] = 0;
      s_aentry[k].seq = nullptr;  // shortcuts hold for one chunk's parallel phase
      s_aentry[k].claim = 0;
    }
    if (threadIdx.x < kDeltaBuckets) s_count[threadIdx.x] = 0;
    if (threadIdx.x == 0) {
      s_run[clen] = seg_begin[c0 + clen];
      s_take = 0;
    }
    __syncthreads();
    for (int j = threadIdx.x; j < clen; j += blockDim.x) {
      const int64_t i = c0 + j;
      const int64_t g0 = seg_begin[i], g1 = seg_begin[i + 1];
      s_run[j] = g0;
      int32_t b = 0;  // empty sequences: bucket 0
      int64_t n = 0;
      for (int64_t g = g0; g < g1; ++g) {
        if (n == 0 && seg_len[g] > 0) b = bucket_of(pool[seg_off[g]]);
        n += seg_len[g];
      }
      s_bucket[j] = (int8_t)b;
      uint8_t fl = done[i] || (kParts && b % nparts != part) ? F_DONE : 0;  // another CTA's op: done here
      if (!fl && !s_stop[b]) {
        int32_t anchor, next_tok;
        find_anchor(t, root, seg_off, seg_len, pool, g0, g1, n, anchor, next_tok);
        if (anchor >= 0) {
          uint32_t h = (uint32_t)(((uint64_t)((uint32_t)anchor * 2654435761u) * kAnchorSlots) >> 32);
          int slot = -1;
          for (int it = 0; it < kAnchorSlots; ++it, h = h + 1 == kAnchorSlots ? 0 : h + 1) {
            const int prev = atomicCAS(&s_akey[h], -1, anchor);
            if (prev == -1 || prev == anchor) {
              slot = (int)h;
              break;
            }
          }
          if (slot >= 0) {
            atomicAdd(op[i] == P2P_OP_INSERT ? &s_ains[slot] : &s_adel[slot], 1);
            s_anchor[j] = anchor;
            s_aslot[j] = (int16_t)slot;
            s_next[j] = next_tok;
            fl |= F_ANCHORED;
          }
        }
      }
      s_flag[j] = fl;
    }
    __syncthreads();
    // 2. Anchors that qualify: at least 3 children whatever this chunk's deletes under them do, and a table
    //    with room for this chunk's inserts under them (grown here if needed).  One warp per anchor.
    for (int k = warp; k < kAnchorSlots; k += kDeltaWarps) {
      const int key = s_akey[k];
      if (key < 0) continue;
      int4 rec = __ldcg(t.node + key);
      bool ok = (int64_t)rec.z - s_adel[k] >= 3;
      if (ok && s_ains[k] > 0) ok = ensure_room(t, key, rec, s_ains[k], lane);
      if (lane == 0) s_aok[k] = ok;
    }
    __syncthreads();
    for (int j = threadIdx.x; j < clen; j += blockDim.x) {
      uint8_t fl = s_flag[j];
      if ((fl & F_ANCHORED) && !s_aok[s_aslot[j]]) s_flag[j] = fl = (uint8_t)(fl & ~F_ANCHORED);
      if (fl & F_ANCHORED) {
        const int a = s_aslot[j];
        const int32_t sb = sub_bucket_of(s_anchor[j], s_next[j], s_ains[a] + s_adel[a] >= kSplitOps);
        s_next[j] = sb;  // from here on: the op's sub-bucket
        atomicAdd(&s_count[sb], 1);
      }
    }
    __syncthreads();
    if (warp == 0) rank_buckets(s_count, s_order, lane);
    __syncthreads();
    // 3. Parallel phase: the warps take sub-buckets of anchored ops, heaviest first.  (Each warp's anchor
    //    shortcut is cleared first: an anchor's table may have grown in step 2.)
    for (;;) {
      int idx = 0;
      if (lane == 0) idx = atomicAdd(&s_take, 1);
      idx = __shfl_sync(kFull, idx, 0);
      if (idx >= kDeltaBuckets) break;
      const int sb = s_order[idx];
      if (s_count[sb] == 0) continue;
      bool stopped = false;
      for (int j0 = 0; j0 < clen; j0 += 32) {
        const int j = j0 + lane;
        unsigned mine = __ballot_sync(kFull, j < clen && (s_flag[j] & (F_ANCHORED | F_DONE)) == F_ANCHORED &&
                                                  s_next[j] == sb);
        while (mine) {
          const int jj = j0 + (__ffs(mine) - 1);
          mine &= mine - 1;
          if (stopped) {  // ops held back behind a stopped op: hold back their first-token buckets too
            if (lane == 0) s_stop[s_bucket[jj]] = 1;
            continue;
          }
          const int64_t i = c0 + jj;
          if (mine) prefetch_op(op, seg_off, seg_len, s_run, c0, j0 + (__ffs(mine) - 1), lane);
          const int r = apply_op(t, root, s_anchor[jj], op[i], s_run[jj], s_run[jj + 1], seg_off, seg_len, pool,
                                 buf, lane, memo, &s_aentry[s_aslot[jj]]);
          if (lane == 0) {
            if (r == OP_DONE) {
              done[i] = 1;
              s_flag[jj] |= F_DONE;
            } else if (r == OP_DEFER) {
              s_flag[jj] |= F_DEFERRED;
            } else {
              s_stop[s_bucket[jj]] = 1;
              if (r == OP_CORRUPT) atomicOr(&gs->status, DELTA_CORRUPT);
            }
          }
          stopped = stopped || (r != OP_DONE && r != OP_DEFER);
          __syncwarp();
        }
      }
    }
    __syncthreads();
    // 4. Serial phase: the warps take first-token buckets of the other ops, heaviest first.
    if (threadIdx.x < kDeltaBuckets) s_count[threadIdx.x] = 0;
    if (threadIdx.x == 0) s_take = 0;
    __syncthreads();
    for (int j = threadIdx.x; j < clen; j += blockDim.x) {
      const uint8_t fl = s_flag[j];
      if (!(fl & F_DONE) && (!(fl & F_ANCHORED) || (fl & F_DEFERRED))) atomicAdd(&s_count[s_bucket[j]], 1);
    }
    __syncthreads();
    if (warp == 0) rank_buckets(s_count, s_order, lane);
    __syncthreads();
    for (;;) {
      int idx = 0;
      if (lane == 0) idx = atomicAdd(&s_take, 1);
      idx = __shfl_sync(kFull, idx, 0);
      if (idx >= kDeltaBuckets) break;
      const int bk = s_order[idx];
      if (s_count[bk] == 0 || *(volatile int*)&s_stop[bk]) continue;
      bool stopped = false;
      for (int j0 = 0; j0 < clen && !stopped; j0 += 32) {
        const int j = j0 + lane;
        bool mine_op = false;
        if (j < clen) {
          const uint8_t fl = s_flag[j];
          mine_op = s_bucket[j] == bk && !(fl & F_DONE) && (!(fl & F_ANCHORED) || (fl & F_DEFERRED));
        }
        unsigned mine = __ballot_sync(kFull, mine_op);
        while (mine && !stopped) {
          const int jj = j0 + (__ffs(mine) - 1);
          mine &= mine - 1;
          const int64_t i = c0 + jj;
          if (mine) prefetch_op(op, seg_off, seg_len, s_run, c0, j0 + (__ffs(mine) - 1), lane);
          const int r = apply_op(t, root, -1, op[i], s_run[jj], s_run[jj + 1], seg_off, seg_len, pool, buf, lane,
                                 memo, nullptr);
          if (lane == 0) {
            if (r == OP_DONE) {
              done[i] = 1;
              s_flag[jj] |= F_DONE;
            } else {
              s_stop[bk] = 1;
              if (r != OP_NEED) atomicOr(&gs->status, DELTA_CORRUPT);
            }
          }
          stopped = r != OP_DONE;
          __syncwarp();
        }
      }
    }
    __syncthreads();
  }
  if (lane < 3) add_stale(t, lane, t.slab[lane].y);  // the rest of this warp's slabs
}

// Validates a device-resident delta into header (int32 words: [0..1] longest sequence as u64, [2] error
// bits STATIC_*, [3] most pool runs of one op); the header must be zero on entry.
__global__ void validate_kernel(int32_t* header, const int32_t* __restrict__ op, const int64_t* __restrict__ seg_begin,
                                const int64_t* __restrict__ seg_off, const int32_t* __restrict__ seg_len, int64_t n,
                                int64_t n_segs, int64_t n_pool, const int64_t* __restrict__ peer_begin, int32_t P) {
  unsigned long long* max_len = reinterpret_cast<unsigned long long*>(header);
  int32_t* err = header + 2;
  int32_t* max_runs = header + 3;
  // Each thread keeps its own maxima and error bits; the warp reduces them and one lane updates the header,
  // so a delta of millions of ops makes a few thousand atomics, not millions on two words.
  unsigned long long my_len = 0;
  int32_t my_runs = 0, my_bits = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    int bits = 0;
    if (op[i] != P2P_OP_INSERT && op[i] != P2P_OP_DELETE) bits |= STATIC_BAD_OP;
    const int64_t a = seg_begin[i], b = seg_begin[i + 1];
    if (a < 0 || b < a || b > n_segs || (i == 0 && a != 0) || (i == n - 1 && b != n_segs)) {
      bits |= STATIC_BAD_SEGMENT;
    } else {
      int64_t len = 0;
      for (int64_t g = a; g < b; ++g) {
        const int64_t off = seg_off[g], l = seg_len[g];
        if (l < 0 || off < 0 || off > n_pool - l) {
          bits |= STATIC_BAD_SEGMENT;
          break;
        }
        len += l;
      }
      if (len > INT32_MAX) bits |= STATIC_TOO_LONG;
      my_len = max(my_len, (unsigned long long)len);
      my_runs = max(my_runs, (int32_t)min(b - a, (int64_t)INT32_MAX));
    }
    my_bits |= bits;
  }
  for (int o = 16; o > 0; o >>= 1) {
    my_len = max(my_len, __shfl_xor_sync(kFull, my_len, o));
    my_runs = max(my_runs, __shfl_xor_sync(kFull, my_runs, o));
    my_bits |= __shfl_xor_sync(kFull, my_bits, o);
  }
  if ((threadIdx.x & 31) == 0) {
    if (my_len) atomicMax(max_len, my_len);
    if (my_runs) atomicMax(max_runs, my_runs);
    if (my_bits) atomicOr(err, my_bits);
  }
  if (peer_begin && blockIdx.x == 0) {
    for (int32_t p = threadIdx.x; p <= P; p += blockDim.x) {
      const int64_t v = peer_begin[p];
      if ((p == 0 && v != 0) || (p == P && v != n) || (p > 0 && v < peer_begin[p - 1]))
        atomicOr(err, STATIC_BAD_PEER_BEGIN);
    }
  }
}

// After a launch that stopped for room: for each tree flagged DELTA_NEED_SPACE, the room its ops not yet
// applied may take -- every remaining INSERT's whole sequence as new label tokens, and the number of those
// INSERTs -- so that the host grows the tree once for the rest of the call instead of once per doubling.
// room[2 * i] = tokens, room[2 * i + 1] = INSERTs (0 for a tree that did not stop).  One CTA per tree.
__global__ void room_kernel(const TreeState* __restrict__ states, const uint8_t* __restrict__ done,
                            const int32_t* __restrict__ op, const int64_t* __restrict__ seg_begin,
                            const int32_t* __restrict__ seg_len, long long* room) {
  const TreeState& s = states[blockIdx.x];
  long long tokens = 0, inserts = 0;
  if (s.status & DELTA_NEED_SPACE) {
    for (int64_t i = s.op_begin + threadIdx.x; i < s.op_end; i += blockDim.x) {
      if (done[i] || op[i] != P2P_OP_INSERT) continue;
      for (int64_t g = seg_begin[i]; g < seg_begin[i + 1]; ++g) tokens += seg_len[g];
      inserts += 1;
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    tokens += __shfl_xor_sync(kFull, tokens, o);
    inserts += __shfl_xor_sync(kFull, inserts, o);
  }
  __shared__ long long s_sum[2][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) {
    s_sum[0][warp] = tokens;
    s_sum[1][warp] = inserts;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    long long a = 0, b = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
      a += s_sum[0][w];
      b += s_sum[1][w];
    }
    room[2 * blockIdx.x] = a;
    room[2 * blockIdx.x + 1] = b;
  }
}

// Sets each tree's op range for this call on the device (peer_begin stays in device memory).
__global__ void init_ranges_kernel(TreeState* states, int32_t nt, const int64_t* __restrict__ peer_begin, int64_t n) {
  const int32_t i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= nt) return;
  states[i].op_begin = peer_begin ? peer_begin[i] : 0;
  states[i].op_end = peer_begin ? peer_begin[i + 1] : n;
  states[i].status = DELTA_OK;
  states[i].need_node = states[i].need_child = states[i].need_label = states[i].need_root = 0;
  states[i].n_absent = 0;
}


constexpr int kCompactThreads = 512;   // two CTAs per SM: every tree of a 256-tree router at once
constexpr int kSmallBits = 4;   // tables of at most 16 slots are copied by one thread
constexpr int kSlotBatch = 4;   // slots of a small table a thread loads before it handles them
constexpr int kUnitSlots = 1024;  // slots of a big table per unit of warp work
constexpr int kUnitCap = 2048;    // units queued per level (a table whose units do not fit is copied by a thread)
constexpr int kLabelThreads = 256;  // compact_labels_kernel: CTAs of 8 warps, a warp per 32 new nodes
constexpr int kLabelCtasPerSm = 8;

struct CompactShared {
  int node, child, label, fail, nunits;
  int2 units[kUnitCap];  // (new node id, first slot) of kUnitSlots slots of a big table; id -1: none
};

// Copies the table of node cid (old record rec) into a fresh table of the same size, one thread.  The
// slots are loaded kSlotBatch at a time; each batch takes its new ids and label space with one reservation,
// and the thread places its entries by linear probing on a bit mask of the slots it has filled, so the new
// table is written once, with no read-back.  Labels are not copied here: each child's scratch entry
// records where its label moves, and compact_labels_kernel moves them all afterwards.
__device__ void compact_node_thread(CompactJob& J, CompactShared& S, int32_t cid, const int4& rec) {
  const int32_t bits = tab_bits(rec.y);
  int32_t noff = 0, live = 0;
  if (bits) {
    const int32_t size = 1 << bits;
    const uint32_t mask = (uint32_t)size - 1;
    noff = atomicAdd(&S.child, size);
    if ((int64_t)noff + size > J.cap_child) {
      atomicOr(&S.fail, 1);
      return;
    }
    uint32_t used = 0;
    for (int32_t j0 = 0; j0 < size; j0 += kSlotBatch) {
      int4 e[kSlotBatch];
#pragma unroll
      for (int u = 0; u < kSlotBatch; ++u)
        e[u] = j0 + u < size ? __ldg(J.child + rec.x + j0 + u) : make_int4(0, 0, 0, 0);
      int32_t cnt = 0, tot = 0;
#pragma unroll
      for (int u = 0; u < kSlotBatch; ++u)
        if (e[u].y >= 1) {
          ++cnt;
          tot += e[u].z >= 0 ? e[u].w : 0;
        }
      if (!cnt) continue;
      int32_t c = atomicAdd(&S.node, cnt);
      int32_t nz = tot ? atomicAdd(&S.label, tot) : 0;
      if ((int64_t)c + cnt > J.cap_node || (int64_t)nz + tot > J.cap_label) {
        atomicOr(&S.fail, 1);
        return;
      }
#pragma unroll
      for (int u = 0; u < kSlotBatch; ++u) {
        if (e[u].y < 1) continue;
        const bool own = e[u].z >= 0;
        const int32_t z = own ? nz : e[u].z;
        J.queue[c] = make_int4(e[u].y, e[u].z, z, own ? e[u].w : 0);
        uint32_t sl = slot_hash(e[u].x, bits);
        while ((used >> sl) & 1u) sl = (sl + 1) & mask;
        used |= 1u << sl;
        J.nchild[noff + sl] = make_int4(e[u].x, c, z, e[u].w);
        ++c;
        nz += own ? e[u].w : 0;
        ++live;
      }
    }
    for (int32_t j = 0; j < size; ++j)
      if (!((used >> j) & 1u)) J.nchild[noff + j] = make_int4(0, 0, 0, 0);
  }
  J.nnode[cid] = make_int4(noff, make_meta(bits, live), rec.z, rec.w);
}

// Copies slots [start, end) of a big table (old record rec) into its new table at noff, one warp: lane j
// takes slot base + j, and new ids and label space for the live slots come from one reservation per 32
// slots (ranks and a prefix sum of label lengths); entries go into the new table with a 64-bit
// compare-and-swap, since other warps fill other ranges of the same table.  As for small tables, the
// labels themselves move later.
__device__ void compact_range_warp(CompactJob& J, CompactShared& S, const int4& rec, int32_t noff, int32_t start,
                                   int32_t end, int lane) {
  const int32_t bits = tab_bits(rec.y);
  const uint32_t mask = (1u << bits) - 1;
  for (int32_t base = start; base < end; base += 32) {
    const int32_t j = base + lane;
    const int4 e = j < end ? __ldg(J.child + rec.x + j) : make_int4(0, 0, 0, 0);
    const bool is_live = j < end && e.y >= 1;
    const unsigned m = __ballot_sync(kFull, is_live);
    if (!m) continue;
    const int32_t cnt = __popc(m), rank = __popc(m & ((1u << lane) - 1));
    const int32_t w = is_live && e.z >= 0 ? e.w : 0;
    int32_t incl = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t y = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += y;
    }
    const int32_t total = __shfl_sync(kFull, incl, 31);
    int32_t lbase = 0, nbase = 0, bad = 0;
    if (lane == 0) {
      lbase = atomicAdd(&S.label, total);
      nbase = atomicAdd(&S.node, cnt);
      bad = (int64_t)lbase + total > J.cap_label || (int64_t)nbase + cnt > J.cap_node;
      if (bad) atomicOr(&S.fail, 1);
    }
    if (__shfl_sync(kFull, bad, 0)) return;
    lbase = __shfl_sync(kFull, lbase, 0);
    nbase = __shfl_sync(kFull, nbase, 0);
    if (is_live) {
      const int32_t cid = nbase + rank;
      const int32_t nz = e.z >= 0 ? lbase + incl - w : e.z;
      J.queue[cid] = make_int4(e.y, e.z, nz, w);
      const unsigned long long kv = (unsigned long long)(uint32_t)e.x | ((unsigned long long)(uint32_t)cid << 32);
      uint32_t sl = slot_hash(e.x, bits);
      for (uint32_t it = 0; it <= mask; ++it, sl = (sl + 1) & mask) {
        if (atomicCAS((unsigned long long*)&J.nchild[noff + sl], 0ull, kv) == 0ull) {
          J.nchild[noff + sl].z = nz;
          J.nchild[noff + sl].w = e.w;
          break;
        }
      }
    }
  }
}

// One CTA per tree: level-synchronous breadth-first copy of the structure from the root.  New ids are
// handed out level by level, so the nodes of the next level are the ids [end, S.node) and the scratch
// entry of id c (old id, old and new label offsets, own-arena label length) is written by the parent's
// copy.  A thread takes each node of the level.  A node whose table has more than 2^kSmallBits slots gets
// its new table range and record from that thread, and its slots are cut into units of kUnitSlots that all
// warps then zero and fill; smaller tables are copied by the thread.  A big table's record counts its
// children from the old record (the live-child count), so no pass has to count them.
__global__ void __launch_bounds__(kCompactThreads) compact_kernel(CompactJob* jobs) {
  CompactJob& J = jobs[blockIdx.x];
  __shared__ CompactShared S;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  constexpr int kWarps = kCompactThreads / 32;
  if (threadIdx.x == 0) {
    S.node = 1;
    S.child = 0;
    S.label = 0;
    S.fail = 0;
    S.nunits = 0;
    J.queue[0] = make_int4(0, 0, 0, 0);
  }
  __syncthreads();
  int begin = 0, end = 1;
  while (begin < end) {
    for (int cid = begin + threadIdx.x; cid < end; cid += kCompactThreads) {
      const int4 rec = __ldg(J.node + J.queue[cid].x);
      const int32_t bits = tab_bits(rec.y);
      if (bits > kSmallBits) {
        const int32_t size = 1 << bits, nu = (size + kUnitSlots - 1) / kUnitSlots;
        const int u0 = atomicAdd(&S.nunits, nu);
        if (u0 + nu <= kUnitCap) {
          const int32_t noff = atomicAdd(&S.child, size);
          if ((int64_t)noff + size > J.cap_child) {
            atomicOr(&S.fail, 1);
            for (int k = 0; k < nu; ++k) S.units[u0 + k] = make_int2(-1, 0);
            continue;
          }
          J.nnode[cid] = make_int4(noff, make_meta(bits, rec.z), rec.z, rec.w);
          for (int k = 0; k < nu; ++k) S.units[u0 + k] = make_int2(cid, k * kUnitSlots);
          continue;
        }
        for (int k = u0; k < kUnitCap; ++k) S.units[k] = make_int2(-1, 0);  // no room: this thread copies it
      }
      compact_node_thread(J, S, cid, rec);
    }
    __syncthreads();
    const int nunits = min(S.nunits, kUnitCap);
    for (int k = warp; k < nunits; k += kWarps) {  // zero every unit's slots first: inserts may wrap into them
      const int2 u = S.units[k];
      if (u.x < 0) continue;
      const int4 nrec = J.nnode[u.x];
      const int32_t n = min(kUnitSlots, (1 << tab_bits(nrec.y)) - u.y);
      for (int32_t j = lane; j < n; j += 32) J.nchild[nrec.x + u.y + j] = make_int4(0, 0, 0, 0);
    }
    __syncthreads();
    for (int k = warp; k < nunits; k += kWarps) {
      const int2 u = S.units[k];
      if (u.x < 0 || __shfl_sync(kFull, *(volatile int*)&S.fail, 0)) continue;
      const int4 rec = __ldg(J.node + J.queue[u.x].x);
      const int32_t noff = J.nnode[u.x].x;
      compact_range_warp(J, S, rec, noff, u.y, min(u.y + kUnitSlots, 1 << tab_bits(rec.y)), lane);
    }
    __syncthreads();
    if (threadIdx.x == 0) S.nunits = 0;
    begin = end;
    end = *(volatile int*)&S.fail ? end : *(volatile int*)&S.node;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    J.n_node = S.node;
    J.n_child = S.child;
    J.n_label = S.label;
    J.status = S.fail;
  }
}

// Moves the own-arena labels of every compacted tree, after compact_kernel: a warp takes 32 consecutive
// new ids of one job, whose scratch entries give each label's old and new offsets and length, and copies
// the labels with all 32 lanes, kLabelsInFlight labels at a time, kLabelSteps coalesced loads per lane
// and label in flight (most own-arena labels are under 128 tokens: one round).  Items are (job, group
// of 32 ids), grid-strided, so one big tree's labels spread over the whole GPU.
constexpr int kLabelSteps = 4;
constexpr int kLabelsInFlight = 4;
__global__ void __launch_bounds__(kLabelThreads) compact_labels_kernel(const CompactJob* __restrict__ jobs,
                                                                       int64_t n_items, int32_t groups_per_job) {
  const int lane = threadIdx.x & 31;
  const int64_t n_warps = (int64_t)gridDim.x * (kLabelThreads / 32);
  for (int64_t it = ((int64_t)blockIdx.x * kLabelThreads + threadIdx.x) >> 5; it < n_items; it += n_warps) {
    const CompactJob& J = jobs[it / groups_per_job];
    const int32_t c0 = (int32_t)(it % groups_per_job) * 32;
    if (J.status != 0 || c0 >= J.n_node) continue;
    const int32_t c = c0 + lane;
    const int4 s = c < J.n_node ? J.queue[c] : make_int4(0, 0, 0, 0);
    const int32_t* __restrict__ src = J.label;
    int32_t* __restrict__ dst = J.nlabel;
    for (int k = 0; k < 32; k += kLabelsInFlight) {
      int32_t y[kLabelsInFlight], z[kLabelsInFlight], w[kLabelsInFlight];
      int32_t wmax = 0;
#pragma unroll
      for (int q = 0; q < kLabelsInFlight; ++q) {
        y[q] = __shfl_sync(kFull, s.y, k + q);
        z[q] = __shfl_sync(kFull, s.z, k + q);
        w[q] = __shfl_sync(kFull, s.w, k + q);
        wmax = max(wmax, w[q]);
      }
      for (int32_t b0 = 0; b0 < wmax; b0 += 32 * kLabelSteps) {
        int32_t x[kLabelsInFlight][kLabelSteps];
#pragma unroll
        for (int q = 0; q < kLabelsInFlight; ++q)
#pragma unroll
          for (int u = 0; u < kLabelSteps; ++u) {
            const int32_t t = b0 + u * 32 + lane;
            x[q][u] = t < w[q] ? __ldg(src + y[q] + t) : 0;
          }
#pragma unroll
        for (int q = 0; q < kLabelsInFlight; ++q)
#pragma unroll
          for (int u = 0; u < kLabelSteps; ++u) {
            const int32_t t = b0 + u * 32 + lane;
            if (t < w[q]) dst[z[q] + t] = x[q][u];
          }
      }
    }
  }
}

__global__ void set_tree_kernel(TreeState* st, TreeView* view, TreeState v, const int32_t* shared) {
  *st = v;
  const int4 root = v.node[0];
  *view = TreeView{v.node, v.child, v.label, shared, v.rfilter, root.x, tab_bits(root.y)};
}

__global__ void refresh_views_kernel(const TreeState* st, TreeView* view, int32_t n, const int32_t* shared) {
  const int32_t i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) {
    const int4 root = st[i].node[0];
    view[i] = TreeView{st[i].node, st[i].child, st[i].label, shared, st[i].rfilter, root.x, tab_bits(root.y)};
  }
}

}  // namespace

cudaError_t launch_refresh_views(const TreeState* d_states, TreeView* d_views, int32_t n, const int32_t* shared,
                                 cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  P2P_TIMED(K_REFRESH_VIEWS, st, (refresh_views_kernel<<<(n + 127) / 128, 128, 0, st>>>(d_states, d_views, n, shared)));
  return cudaGetLastError();
}

cudaError_t launch_compact(CompactJob* d_jobs, int32_t n_jobs, int32_t max_cap_node, int num_sms, cudaStream_t st) {
  if (n_jobs <= 0) return cudaSuccess;
  P2P_TIMED(K_COMPACT, st, (compact_kernel<<<n_jobs, kCompactThreads, 0, st>>>(d_jobs)));
  const int32_t groups = (max_cap_node + 31) / 32;
  P2P_TIMED(K_COMPACT_LABELS, st,
            (compact_labels_kernel<<<std::max(num_sms, 1) * kLabelCtasPerSm, kLabelThreads, 0, st>>>(
                d_jobs, (int64_t)n_jobs * groups, groups)));
  return cudaGetLastError();
}

cudaError_t launch_delta(TreeState* d_states, uint8_t* done, int32_t n_trees, const int32_t* op,
                         const int64_t* seg_begin, const int64_t* seg_off, const int32_t* seg_len, const int32_t* pool,
                         int32_t* gather, int64_t gather_stride, const int32_t* shared, cudaStream_t st,
                         const GlobalMemo* gm, const int32_t* parts, int32_t n_blocks) {
  if (n_trees <= 0) return cudaSuccess;
  const int dyn = delta_smem_bytes();
  cudaError_t e = cudaFuncSetAttribute(parts ? delta_kernel<true> : delta_kernel<false>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
  if (e != cudaSuccess) return e;
  if (parts) {
    P2P_TIMED(K_DELTA, st,
              (delta_kernel<true><<<n_blocks, kDeltaWarps * 32, dyn, st>>>(
                  d_states, done, op, seg_begin, seg_off, seg_len, pool, gather, gather_stride, shared,
                  gm ? gm->keys : nullptr, gm ? gm->vals : nullptr, gm ? gm->mask : 0u, parts)));
  } else {
    P2P_TIMED(K_DELTA, st,
              (delta_kernel<false><<<n_trees, kDeltaWarps * 32, dyn, st>>>(
                  d_states, done, op, seg_begin, seg_off, seg_len, pool, gather, gather_stride, shared,
                  gm ? gm->keys : nullptr, gm ? gm->vals : nullptr, gm ? gm->mask : 0u, nullptr)));
  }
  return cudaGetLastError();
}

cudaError_t launch_validate(int32_t* header, const p2p_delta* d, int32_t peer, int32_t P, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(header, 0, kStaticHeaderInts * sizeof(int32_t), st);
  if (e != cudaSuccess) return e;
  const p2p_seqs& S = d->seqs;
  const int64_t blocks = std::min<int64_t>((S.n + 255) / 256, 4096);
  P2P_TIMED(K_VALIDATE, st,
            (validate_kernel<<<(int)std::max<int64_t>(blocks, 1), 256, 0, st>>>(
                header, d->op, S.seg_begin, S.seg_off, S.seg_len, S.n, S.n_segs, S.n_pool,
                peer == -1 ? d->peer_begin : nullptr, P)));
  return cudaGetLastError();
}

cudaError_t launch_room(const TreeState* d_states, int32_t nt, const uint8_t* done, const int32_t* op,
                        const int64_t* seg_begin, const int32_t* seg_len, long long* room, cudaStream_t st) {
  if (nt <= 0) return cudaSuccess;
  P2P_TIMED(K_ROOM, st, (room_kernel<<<nt, 256, 0, st>>>(d_states, done, op, seg_begin, seg_len, room)));
  return cudaGetLastError();
}

cudaError_t launch_init_ranges(TreeState* d_states, int32_t nt, const int64_t* peer_begin, int64_t n, cudaStream_t st) {
  P2P_TIMED(K_INIT_RANGES, st, (init_ranges_kernel<<<(nt + 127) / 128, 128, 0, st>>>(d_states, nt, peer_begin, n)));
  return cudaGetLastError();
}

cudaError_t launch_set_tree(TreeState* d_state, TreeView* d_view, TreeState value, const int32_t* shared,
                            cudaStream_t st) {
  P2P_TIMED(K_SET_TREE, st, (set_tree_kernel<<<1, 1, 0, st>>>(d_state, d_view, value, shared)));
  return cudaGetLastError();
}

}  // namespace p2p
