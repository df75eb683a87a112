// route_kernel.cu -- batched longest-prefix match against P radix trees and the route decision.
//
// Computes, for every request r_b and tree T_p, match(r_b, T_p) = PrefixMatch of Algorithm 1 (the
// number of leading request tokens found along one path of T_p, a partial edge included), and the
// chosen peer argmax_p (match - alpha*load_p, -load_p, -p) (Algorithm 1's argmax with a load term).
//
// Passes.  A grouped batch (group_kernel.cu) is routed by a leader pass and a follower pass.  Leaders of
// short requests, and all followers, are walked by lane_kernel (a lane per tree; below).  Leaders whose
// requests are longer than a staging window on average go to route_kernel:
//
// route_kernel schedule.  A CTA takes requests b = list[blockIdx.x], list[blockIdx.x + gridDim.x], ...; its
// work items are (request, group of G consecutive trees) in that order, handed to warps from a shared
// counter, so a warp that finishes short walks immediately takes the next item.  Requests are staged in
// shared memory in kSlots slots: the warp that takes a request's first item copies its tokens in with one
// bulk (TMA) copy (up to kSlotTokens; longer requests read the rest through the read-only path); warps with
// later items of that request wait until it is staged; the last warp to finish one of its items writes the
// route and frees the slot for the request kSlots later.  Every wait is bounded.
//
// A warp-cooperative walk: a child lookup probes 32 slots of the node's children hash table at once (one
// coalesced load, whatever the fan-out), and an edge label is compared 32 consecutive tokens per warp load,
// up to kUnroll loads in flight per lane, folded into one vote per block; the first mismatch is searched
// only inside the block that holds it.  The route decision keeps the max of a packed 64-bit key per
// request.  decide_kernel (p2p_route_decide) makes the decision again from a match matrix with some trees
// excluded and also returns the next-best tree (Sections 3.2 and 3.3).  Integer work only: no tensor cores.
#include "internal.h"

namespace p2p {
namespace {

constexpr int kWarps = 16;              // warps per CTA
constexpr int kThreads = kWarps * 32;
constexpr int kSlots = 4;               // requests staged at a time per CTA
constexpr int kSlotTokens = 4096;       // tokens of a request kept in shared memory (16 KB per slot)
constexpr int kCtasPerSm = 2;           // 32 warps per SM: 64 KB of slots and <= 64 registers per thread
constexpr int kUnroll = 16;             // label loads in flight per lane on long labels (512 tokens per step)
constexpr int kMaxGroup = 8;            // trees per work item, at most
constexpr unsigned kFull = 0xffffffffu;
constexpr int kSpinLimit = 1 << 24;     // bounded waits (~1 s): the kernel flags ERR_STALL and stops

struct Slot {
  unsigned long long bar;   // mbarrier of the slot's bulk copy (one phase per staged request)
  unsigned long long best;  // max packed route key so far
  long long len;    // request length; -1 = the request's offsets are invalid
  long long start;  // index of the request's first token in `tokens`
  int ready;        // request (CTA-local index k) whose tokens are staged here
  int free_for;     // the request allowed to stage here next
  int len_s;        // tokens held in shared memory
  int shift;        // token j of the request sits at slot token shift + j (keeps bulk copies 16-byte aligned)
  int done;         // items of the request finished
  int row;          // grouped batch: the leader's checkpoint row (-1: none)
  int climit;       // grouped batch: checkpoints are taken at positions <= climit
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

// Bulk copy global -> shared (untiled TMA), completing on the slot's mbarrier.
__device__ __forceinline__ void bulk_copy(void* dst, const void* src, uint32_t bytes, unsigned long long* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               :: "r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect(unsigned long long* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" :: "r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_test(unsigned long long* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
               : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
  return ok != 0;
}

__device__ __forceinline__ int32_t req_at(const int32_t* s_req, int32_t n_s, const int32_t* g_req, int32_t i) {
  return i < n_s ? s_req[i] : __ldg(g_req + i);
}

// Child with first token `tok` in the children table of 2^bits slots at tab: one coalesced probe of 32
// consecutive slots (a table is at most 1/2 full, so the probe run almost always fits).  Returns false if
// there is no such child.
__device__ __forceinline__ bool find_child(const int4* __restrict__ tab, int32_t bits, int32_t tok, int lane,
                                           int4& out) {
  if (bits == 0) return false;
  const uint32_t mask = (1u << bits) - 1, h = slot_hash(tok, bits);
  for (uint32_t base = 0; base <= mask; base += 32) {
    const int4 e = __ldg(tab + ((h + base + lane) & mask));
    const unsigned live = __ballot_sync(kFull, e.y >= 1 && e.x == tok);
    const unsigned empty = __ballot_sync(kFull, e.y == 0);
    const int fl = live ? __ffs(live) - 1 : 64;
    const int fe = empty ? __ffs(empty) - 1 : 64;
    if (fl < fe) {
      out.x = tok;
      out.y = __shfl_sync(kFull, e.y, fl);
      out.z = __shfl_sync(kFull, e.z, fl);
      out.w = __shfl_sync(kFull, e.w, fl);
      return true;
    }
    if (fe < 64) return false;
  }
  return false;
}

// Request token j: from the shared-memory window, or past it through the read-only path.
template <bool kGlobal>
__device__ __forceinline__ int32_t rq(const int32_t* req, int32_t j) {
  if constexpr (kGlobal) return __ldg(req + j);
  else return req[j];
}

// U label loads of 32 tokens in flight per lane over [j0, j0 + 32U), a block inside both the label and the
// request.  The block is folded into one OR of XORs per lane and one warp vote; only a block that holds a
// mismatch is searched again for the first one.  Returns it, or -1.  Positions are 32-bit: a walk never
// passes more tokens than one tree path holds (< 2^31).
template <int U, bool kGlobal>
__device__ __forceinline__ int32_t compare_full(const int32_t* __restrict__ lab, const int32_t* req, int32_t j0,
                                                int lane) {
  int32_t v[U];
#pragma unroll
  for (int u = 0; u < U; ++u) v[u] = __ldg(lab + j0 + u * 32 + lane);
  int32_t diff = 0;
#pragma unroll
  for (int u = 0; u < U; ++u) diff |= v[u] ^ rq<kGlobal>(req, j0 + u * 32 + lane);
  if (!__any_sync(kFull, diff != 0)) return -1;
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const unsigned m = __ballot_sync(kFull, v[u] != rq<kGlobal>(req, j0 + u * 32 + lane));
    if (m) return j0 + u * 32 + (__ffs(m) - 1);
  }
  return -1;
}

// As compare_full<4> for a block that may run past end (tokens at or after end are ignored).
template <bool kGlobal>
__device__ __forceinline__ int32_t compare_tail(const int32_t* __restrict__ lab, const int32_t* req, int32_t j0,
                                                int32_t end, int lane) {
  int32_t v[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int32_t j = j0 + u * 32 + lane;
    v[u] = j < end ? __ldg(lab + j) : 0;
  }
  int32_t diff = 0;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int32_t j = j0 + u * 32 + lane;
    if (j < end) diff |= v[u] ^ rq<kGlobal>(req, j);
  }
  if (!__any_sync(kFull, diff != 0)) return -1;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int32_t j = j0 + u * 32 + lane;
    const unsigned m = __ballot_sync(kFull, j < end && v[u] != rq<kGlobal>(req, j));
    if (m) return j0 + u * 32 + (__ffs(m) - 1);
  }
  return -1;
}

// First j in [j0, end) with lab[j] != req[j], or -1.  After one block at j0 the label side continues at a
// 128-byte-aligned position at or below j0 + 32 (re-comparing <= 31 tokens): a warp's 32 consecutive label
// tokens are then one cache line, and its 32 request tokens in shared memory fall in 32 distinct banks at
// any alignment, so each load is a single wavefront on both sides.
template <int U, bool kGlobal>
__device__ __forceinline__ int32_t compare_range(const int32_t* __restrict__ lab, const int32_t* req, int32_t j0,
                                                 int32_t end, int lane) {
  if (j0 + 32 <= end) {
    const int32_t k = compare_full<1, kGlobal>(lab, req, j0, lane);
    if (k >= 0) return k;
    j0 += 32;
    j0 -= (int32_t)(((uintptr_t)(lab + j0) >> 2) & 31);
    for (; j0 + U * 32 <= end; j0 += U * 32) {
      const int32_t k2 = compare_full<U, kGlobal>(lab, req, j0, lane);
      if (k2 >= 0) return k2;
    }
  }
  for (; j0 < end; j0 += 128) {
    const int32_t k = compare_tail<kGlobal>(lab, req, j0, end, lane);
    if (k >= 0) return k;
  }
  return -1;
}

// First j in [from, lim) with lab[j] != request[pos + j], or lim; the tokens before `from` are known to
// match (from >= 1: lab[0] == request[pos] is known).  Request tokens inside the shared-memory window (the
// first n_s) come from it, later ones from global memory.
template <int U>
__device__ __forceinline__ int32_t first_mismatch(const int32_t* __restrict__ lab, const int32_t* s_req, int32_t n_s,
                                                  const int32_t* g_req, int32_t pos, int32_t lim, int32_t from,
                                                  int lane) {
  if (from >= lim) return lim;
  const int32_t split = max(from, min(lim, n_s - pos));
  int32_t k = compare_range<U, false>(lab, s_req + pos, from, split, lane);
  if (k < 0 && split < lim) k = compare_range<U, true>(lab, g_req + pos, split, lim, lane);
  return k < 0 ? lim : k;
}

// match(r, T) for one tree, computed by the whole warp (result uniform across lanes).  len is the request
// length clamped to 2^31 - 1 (no match can be longer than a tree path).  The first `known` tokens are known
// to be matched (known <= match(r, T)): the walk still follows their path but does not compare them.
template <int U>
__device__ int32_t walk_from(const TreeView& t, int4 ce, const int32_t* s_req, int32_t n_s, const int32_t* g_req,
                             int32_t len, int32_t known, int lane, int32_t* err, int32_t climit, int4* ck);

// Checkpoint of a walk at the root: {position 0, the root's table offset, its meta, "has children"}.
__device__ __forceinline__ int4 root_checkpoint(const TreeView& t) {
  return make_int4(0, t.root_off, make_meta(t.root_bits, 0), 1);
}

template <int U>
__device__ int32_t walk(const TreeView& t, const int32_t* s_req, int32_t n_s, const int32_t* g_req, int32_t len,
                        int32_t known, int lane, int32_t* err, int32_t climit, int4* ck) {
  if (len == 0) return 0;
  int4 ce;
  if (!find_child(t.child + t.root_off, t.root_bits, req_at(s_req, n_s, g_req, 0), lane, ce)) return 0;
  return walk_from<U>(t, ce, s_req, n_s, g_req, len, known, lane, err, climit, ck);
}

// The walk below the root, from the root's child entry ce for the request's first token (len >= 1).  If ck
// is not NULL, lane 0 stores there each node boundary the walk reaches at a position <= climit (so the
// deepest one stays): {position, the node's table offset, its meta, its child count}.
template <int U>
__device__ int32_t walk_from(const TreeView& t, int4 ce, const int32_t* s_req, int32_t n_s, const int32_t* g_req,
                             int32_t len, int32_t known, int lane, int32_t* err, int32_t climit, int4* ck) {
  int32_t pos = 0;
  for (;;) {
    if (ce.w <= 0 || ce.y <= 0) {  // cannot happen in a valid tree; keeps the loop finite if it does
      if (lane == 0) atomicOr(err, ERR_CORRUPT_TREE);
      break;
    }
    const int4 nn = __ldg(t.node + ce.y);  // the child's record, fetched while its label is compared
    const int32_t lim = min(ce.w, len - pos);
    const int32_t k = first_mismatch<U>(label_ptr(t.label, t.shared, ce.z), s_req, n_s, g_req, pos, lim,
                                        max(1, known - pos), lane);
    pos += k;
    if (ck && k == ce.w && pos <= climit && lane == 0) *ck = make_int4(pos, nn.x, nn.y, nn.z);
    if (k < ce.w || pos >= len || nn.z <= 0) break;
    if (!find_child(t.child + nn.x, tab_bits(nn.y), req_at(s_req, n_s, g_req, pos), lane, ce)) break;
  }
  return pos;
}

// Lane 0 waits (bounded) until *flag == v; the outcome is broadcast to the warp.
__device__ __forceinline__ bool wait_for(const int* flag, int v, int lane) {
  int ok = 1;
  if (lane == 0) {
    int it = 0;
    while (*(const volatile int*)flag != v && ++it < kSpinLimit) __nanosleep(64);
    ok = it < kSpinLimit;
  }
  return __shfl_sync(kFull, ok, 0) != 0;
}

// Packed route key: (score + 2^31) << 32 | (0xFFFF - load) << 16 | (0xFFFF - p); a larger key is a better
// route (higher score, then lower load, then lower index).  The host guarantees alpha * load <= 2^31 - 1,
// load <= 65535 and P <= 65536, so every field fits.  The staged load word of tree p carries kExcluded when
// the decision with excluded trees takes p out (the load itself is the low 16 bits).
constexpr int32_t kExcluded = kLoadExcluded;
__device__ __forceinline__ unsigned long long route_key(int32_t m, int32_t ld, int32_t p, int32_t alpha) {
  const long long score = (long long)m - (long long)alpha * ld;
  return ((unsigned long long)(score + 2147483648LL) << 32) | ((unsigned long long)(0xFFFF - ld) << 16) |
         (unsigned long long)(0xFFFF - p);
}

// The route decision of one request, accumulated over its trees by one lane and merged over the warp.
//   kDecide = false: the max packed key (the route of Algorithm 1's argmax with the load term).
//   kDecide = true: the two largest keys of the trees not excluded (kExcluded in the load word; Section 3.2,
//   a peer that pushes back; Section 3.3, a suspected-failed peer), i.e. the best target and the next-best one
//   that a request falls back to when forwarding times out.  A key is never 0 (score + 2^31 >= 1), so 0 marks
//   "no candidate" (-1 out).
template <bool kDecide>
struct RouteAcc;
template <>
struct RouteAcc<false> {
  unsigned long long k1 = 0;
  __device__ __forceinline__ void add(int32_t m, int32_t ldw, int32_t p, int32_t alpha) {
    const unsigned long long key = route_key(m, ldw, p, alpha);
    k1 = key > k1 ? key : k1;
  }
  __device__ __forceinline__ void warp_merge() {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long other = __shfl_xor_sync(kFull, k1, o);
      k1 = other > k1 ? other : k1;
    }
  }
  __device__ __forceinline__ void write(int64_t b, int32_t* out_peer, int32_t*) const {
    out_peer[b] = 0xFFFF - (int32_t)(k1 & 0xFFFFull);
  }
};
template <>
struct RouteAcc<true> {
  unsigned long long k1 = 0, k2 = 0;
  __device__ __forceinline__ void add(int32_t m, int32_t ldw, int32_t p, int32_t alpha) {
    if (ldw & kExcluded) return;
    const unsigned long long key = route_key(m, ldw, p, alpha);
    if (key > k1) {
      k2 = k1;
      k1 = key;
    } else if (key > k2) {
      k2 = key;
    }
  }
  // Merges the keys of lane groups of 2 * first lanes (the whole warp by default) into each of their lanes.
  __device__ __forceinline__ void warp_merge(int first = 16) {
#pragma unroll
    for (int o = first; o > 0; o >>= 1) {
      const unsigned long long o1 = __shfl_xor_sync(kFull, k1, o), o2 = __shfl_xor_sync(kFull, k2, o);
      const unsigned long long lo = k1 < o1 ? k1 : o1, hi = k1 < o1 ? o1 : k1, r2 = k2 < o2 ? o2 : k2;
      k1 = hi;
      k2 = lo < r2 ? r2 : lo;
    }
  }
  __device__ __forceinline__ void write(int64_t b, int32_t* out_peer, int32_t* out_next) const {
    out_peer[b] = k1 ? 0xFFFF - (int32_t)(k1 & 0xFFFFull) : -1;
    if (out_next) out_next[b] = k2 ? 0xFFFF - (int32_t)(k2 & 0xFFFFull) : -1;
  }
};

// The lane walks' accumulator.  The plain argmax keeps its key in a register; the decision with excluded
// trees keeps a lane's two keys in shared memory, so the walk loops (at their register limit) do not lose
// loads in flight to it.  finish() merges over the warp and lane 0 writes the decision.
template <bool kDecide>
struct LaneAcc : RouteAcc<false> {
  __device__ explicit LaneAcc(unsigned long long*) {}
  __device__ __forceinline__ void finish(int lane, int64_t b, int32_t* out_peer, int32_t* out_next) {
    warp_merge();
    if (lane == 0) write(b, out_peer, out_next);
  }
};
template <>
struct LaneAcc<true> {
  unsigned long long* s;  // s[0] and s[32]: this lane's largest and second-largest key
  __device__ explicit LaneAcc(unsigned long long* p) : s(p) {
    s[0] = 0;
    s[32] = 0;
  }
  __device__ __forceinline__ void add(int32_t m, int32_t ldw, int32_t p, int32_t alpha) {
    if (ldw & kExcluded) return;
    const unsigned long long key = route_key(m, ldw, p, alpha), k1 = s[0];
    if (key > k1) {
      s[32] = k1;
      s[0] = key;
    } else if (key > s[32]) {
      s[32] = key;
    }
  }
  __device__ __forceinline__ void finish(int lane, int64_t b, int32_t* out_peer, int32_t* out_next) {
    RouteAcc<true> r;
    r.k1 = s[0];
    r.k2 = s[32];
    r.warp_merge();
    if (lane == 0) r.write(b, out_peer, out_next);
  }
};

// Routes the leaders list[0 .. *count) of a grouped batch with full walks.  kDecide: the decision with
// excluded trees and the next-best target (RouteAcc<true>), made by the request's last warp from its match
// row once every item of the request has written its part.
template <bool kDecide>
__global__ void __launch_bounds__(kThreads, kCtasPerSm) route_kernel(
    const TreeView* __restrict__ trees, int32_t P, const int32_t* __restrict__ tokens, int64_t n_tokens,
    int64_t tok_base, const int64_t* __restrict__ offsets, int64_t B, const int32_t* __restrict__ list,
    const int32_t* __restrict__ count, const int32_t* __restrict__ gid, const int32_t* __restrict__ cmin,
    int4* __restrict__ ckpt, const int32_t* __restrict__ load, int32_t alpha, int32_t* __restrict__ out_match,
    int32_t* __restrict__ out_peer, int32_t* err, int32_t* __restrict__ out_next) {
  extern __shared__ __align__(128) int32_t s_tok[];  // kSlots x kSlotTokens
  __shared__ Slot s_slot[kSlots];
  __shared__ int4 s_root[kWarps][32];  // per warp: the item's root-table windows
  __shared__ unsigned long long s_next;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x < kSlots) {
    Slot& sl = s_slot[threadIdx.x];
    sl.ready = -1;
    sl.free_for = threadIdx.x;
    sl.done = 0;
    sl.best = 0;
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" :: "r"(smem_u32(&sl.bar)) : "memory");
  }
  if (threadIdx.x == 0) s_next = 0;
  __syncthreads();
  const int64_t n_all = *count;  // requests of this launch
  const int64_t n_req = n_all > blockIdx.x ? (n_all - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
  // A work item is (request k, trees p0 .. p0 + G - 1): G grows with P so that the per-item costs (the
  // shared counter, the staging waits, the route-key merge) are shared by several walks while every warp of
  // the CTA still finds items of the same request.
  const int32_t G = min(kMaxGroup, max(1, P / kWarps));
  const int32_t C = (P + G - 1) / G;  // work items per request
  const unsigned long long total = (unsigned long long)n_req * (unsigned long long)C;
  const bool small = total <= 0xffffffffull;  // 32-bit item arithmetic (the usual case) is much cheaper
  for (;;) {
    unsigned long long i = 0;
    if (lane == 0) i = atomicAdd(&s_next, 1ull);
    i = __shfl_sync(kFull, i, 0);
    if (i >= total) break;
    int64_t k;
    int32_t c;
    if (small) {
      const uint32_t k32 = (uint32_t)i / (uint32_t)C;
      k = k32;
      c = (int32_t)((uint32_t)i - k32 * (uint32_t)C);
    } else {
      k = (int64_t)(i / (unsigned long long)C);
      c = (int32_t)(i - (unsigned long long)k * C);
    }
    const int s = (int)(k % kSlots);
    const int64_t kb = blockIdx.x + k * gridDim.x;
    const int64_t b = __ldg(list + kb);
    Slot& sl = s_slot[s];
    int32_t* st = s_tok + s * kSlotTokens;
    if (c == 0) {
      // Stage request k once the request kSlots earlier has released the slot.
      if (!wait_for(&sl.free_for, (int)k, lane)) {
        if (lane == 0) atomicOr(err, ERR_STALL);
        return;
      }
      const int64_t start = __ldg(offsets + b) - tok_base, end = __ldg(offsets + b + 1) - tok_base;
      const bool valid = start >= 0 && start <= end && end <= n_tokens;
      const int32_t* g = tokens + (valid ? start : 0);
      // Token j goes to slot token shift + j, so that 16-byte-aligned global addresses land on 16-byte-aligned
      // shared addresses: the aligned middle of the request moves with one bulk copy, the <= 3 tokens on
      // each side with plain loads.
      const int32_t shift = (int32_t)(((uintptr_t)g >> 2) & 3);
      const int32_t n_s = valid ? (int32_t)min(end - start, (int64_t)(kSlotTokens - shift)) : 0;
      const int32_t j_lo = min((4 - shift) & 3, n_s);
      const int32_t j_hi = max(j_lo, n_s - (int32_t)(((uintptr_t)(g + n_s) >> 2) & 3));
      const uint32_t bytes = (uint32_t)(j_hi - j_lo) * 4u;
      if (lane == 0) {
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // earlier reads of the slot come first
        mbar_arrive_expect(&sl.bar, bytes);
        if (bytes) bulk_copy(st + shift + j_lo, g + j_lo, bytes, &sl.bar);
      }
      if (lane < j_lo) st[shift + lane] = __ldg(g + lane);
      if (lane < n_s - j_hi) st[shift + j_hi + lane] = __ldg(g + j_hi + lane);
      // Bounded wait for the bulk copy (this slot's phase parity alternates with each staged request).
      const uint32_t parity = (uint32_t)((k / kSlots) & 1);
      int ok = 1;
      if (lane == 0) {
        int it = 0;
        while (!mbar_test(&sl.bar, parity) && ++it < kSpinLimit) __nanosleep(32);
        ok = it < kSpinLimit;
      }
      if (!__shfl_sync(kFull, ok, 0)) {
        if (lane == 0) atomicOr(err, ERR_STALL);
        return;
      }
      __syncwarp();
      if (lane == 0) {
        sl.len = valid ? end - start : -1;
        sl.start = valid ? start : 0;
        sl.len_s = n_s;
        sl.shift = shift;
        sl.best = 0;
        sl.done = 0;
        sl.row = __ldg(gid + b);
        sl.climit = __ldg(cmin + b);
        __threadfence_block();
        *(volatile int*)&sl.ready = (int)k;
      }
      __syncwarp();
    } else {
      // Wait until request k is staged: its slot fields (ready flag), then its bulk copy (mbarrier phase).
      bool ok = wait_for(&sl.ready, (int)k, lane);
      if (ok && lane == 0) {
        int it = 0;
        while (!mbar_test(&sl.bar, (uint32_t)((k / kSlots) & 1)) && ++it < kSpinLimit) __nanosleep(32);
        ok = it < kSpinLimit;
      }
      if (!__shfl_sync(kFull, (int)ok, 0)) {
        if (lane == 0) atomicOr(err, ERR_STALL);
        return;
      }
      __threadfence_block();
    }
    const int64_t len = *(volatile long long*)&sl.len;
    const int64_t start = *(volatile long long*)&sl.start;
    const int32_t n_s = *(volatile int*)&sl.len_s;
    const int32_t* req = st + *(volatile int*)&sl.shift;
    const int32_t len32 = (int32_t)min(len, (int64_t)INT32_MAX);
    const int32_t p1 = min(P, (c + 1) * G);
    const int32_t row = *(volatile int*)&sl.row, climit = row >= 0 ? *(volatile int*)&sl.climit : -1;
    // The request's first token in the root tables of the item's trees at once: lanes 4i .. 4i+3 read four
    // consecutive slots of tree c*G + i's table (G <= 8).  A tree whose window holds the token before any
    // empty slot starts its walk below the root; one whose window has an empty slot first does not hold
    // the token; one whose window is all other keys probes again in full.
    unsigned hit_mask = 0, empty_mask = 0;
    int4* s_re = s_root[threadIdx.x >> 5];  // this warp's window entries
    if (len > 0) {
      int4 re = make_int4(0, 0, 0, 0);
      const int32_t tp = c * G + (lane >> 2);
      const int32_t tok0 = req_at(req, n_s, tokens + start, 0);
      bool hit = false, empty = false;
      if (tp < p1) {
        const int32_t bits = trees[tp].root_bits;
        if (bits > 0 && root_filter_has(trees[tp].rfilter, tok0)) {
          const uint32_t mask = (1u << bits) - 1;
          re = __ldg(trees[tp].child + trees[tp].root_off + ((slot_hash(tok0, bits) + (lane & 3)) & mask));
          hit = re.y >= 1 && re.x == tok0;
          empty = re.y == 0;
        } else {
          empty = true;  // an empty root table, or a first token the root filter rules out
        }
      }
      s_re[lane] = re;
      __syncwarp();
      hit_mask = __ballot_sync(kFull, hit);
      empty_mask = __ballot_sync(kFull, empty);
    }
    unsigned long long best = 0;
    for (int32_t p = c * G; p < p1; ++p) {
      int32_t m = 0;
      if (len > 0) {
        const int sh = 4 * (p - c * G);
        const unsigned gh = (hit_mask >> sh) & 0xFu, ge = (empty_mask >> sh) & 0xFu;
        const int fh = gh ? __ffs(gh) : 64, fe = ge ? __ffs(ge) : 64;
        int4* ck = nullptr;
        if (row >= 0) {  // the walk overwrites the root checkpoint with deeper boundaries
          ck = ckpt + (int64_t)row * P + p;
          if (lane == 0) *ck = root_checkpoint(trees[p]);
        }
        if (fh < fe) {
          const int4 ce = s_re[sh + fh - 1];  // written by this warp before its ballots
          m = walk_from<kUnroll>(trees[p], ce, req, n_s, tokens + start, len32, 0, lane, err, climit, ck);
        } else if (fe == 64) {
          m = walk<kUnroll>(trees[p], req, n_s, tokens + start, len32, 0, lane, err, climit, ck);
        }
      }
      if (lane == 0) {
        out_match[b * P + p] = m;
        const unsigned long long key = route_key(m, __ldg(load + p), p, alpha);
        best = key > best ? key : best;
      }
    }
    int last = 0;
    if (lane == 0) {
      if (!kDecide) atomicMax(&sl.best, best);
      __threadfence_block();
      last = atomicAdd(&sl.done, 1) == C - 1;  // last item of request k: route it, free the slot
    }
    if (__shfl_sync(kFull, last, 0)) {
      __threadfence_block();
      if (len < 0) {
        if (lane == 0) {
          out_peer[b] = -1;
          if (kDecide && out_next) out_next[b] = -1;
          atomicOr(err, ERR_BAD_OFFSETS);
        }
      } else if constexpr (kDecide) {
        // The row was written by this CTA's warps before their (fenced) item counts: read it past L1.
        RouteAcc<true> acc;
        for (int32_t p = lane; p < P; p += 32) acc.add(__ldcg(out_match + b * P + p), __ldg(load + p), p, alpha);
        acc.warp_merge();
        if (lane == 0) acc.write(b, out_peer, out_next);
      } else if (lane == 0) {
        const unsigned long long bk = *(volatile unsigned long long*)&sl.best;
        out_peer[b] = 0xFFFF - (int32_t)(bk & 0xFFFFull);
      }
      __syncwarp();
      if (lane == 0) {
        __threadfence_block();
        *(volatile int*)&sl.free_for = (int)(k + kSlots);
      }
    }
    __syncwarp();
  }
}

// ---- Lane walks (leaders of short requests, and followers) ----------------------------------------------
//
// A warp takes one request and each lane one tree (lanes j, j + 32, ...), so a warp keeps 32 independent
// chains of dependent loads in flight.  Edges are walked by their lane; a label compare that goes on past
// its first 8 tokens with more than kThreadSpan tokens left is done by the whole warp, once for every lane
// waiting at the same label address and request position.
//   Leaders: whole walks, and the checkpoints their followers resume from.
//   A follower f with leader l and exact common prefix c: in tree p, match(f) = match(l) if match(l) < c,
//   else a walk resumed at the leader's checkpoint that does not compare f's first c tokens.

constexpr int kFollowThreads = 256;
constexpr int kFollowCtasPerSm = 4;
constexpr int kThreadSpan = 64;
constexpr int kFollowIlp = 2;  // trees a follower's lane takes per iteration (their first loads overlap; 3 or 4 spill)

// One thread: the child with first token tok in a table of 2^bits (>= 4, even) slots, two slots per step of
// the linear probe.  Returns false if there is none.
__device__ __forceinline__ bool find_child_1(const int4* __restrict__ tab, int32_t bits, int32_t tok, int4& out) {
  if (bits == 0) return false;
  const uint32_t mask = (1u << bits) - 1, h = slot_hash(tok, bits);
  for (uint32_t i = 0; i <= mask; i += 2) {
    const int4 a = __ldg(tab + ((h + i) & mask));
    const int4 b = __ldg(tab + ((h + i + 1) & mask));
    if (a.y >= 1 && a.x == tok) {
      out = a;
      return true;
    }
    if (a.y == 0) return false;
    if (b.y >= 1 && b.x == tok) {
      out = b;
      return true;
    }
    if (b.y == 0) return false;
  }
  return false;
}

// One thread: first j in [from, lim) with lab[j] != req[j], or lim; 8 token pairs in flight per step.
__device__ __forceinline__ int32_t first_diff_1(const int32_t* __restrict__ lab, const int32_t* __restrict__ req,
                                                int32_t from, int32_t lim) {
  for (int32_t j0 = from; j0 < lim; j0 += 8) {
    int32_t x[8], y[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int32_t j = j0 + u;
      x[u] = j < lim ? __ldg(lab + j) : 0;
      y[u] = j < lim ? __ldg(req + j) : 0;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (j0 + u < lim && x[u] != y[u]) return j0 + u;
  }
  return lim;
}

// Advances the walks of a warp's lanes edge by edge until none is left (collective: every lane of the warp
// calls it).  Lane state: tree p, the edge ce to walk at position pos (act), m = tokens matched so far,
// known = tokens known to match without comparing, and for leaders the checkpoint slot ck (NULL: none)
// with the deepest position climit it records.  A lane compares an edge's label itself when it leaves
// within the first kFirst tokens or the edge has at most kThreadSpan tokens left; longer compares are done
// by the whole warp, once per distinct (label address, request position): the long prompt prefixes are
// interned labels shared by many trees, so one compare serves every lane at that label.  Leaders take
// kFirst = 8.  Followers of a batch of requests shorter than a staging window on average take 16: they
// resume past the shared prefix, where labels tend to end within a few tokens (the scale workload's follower
// pass 5.0 -> 4.8 ms); followers of long requests take 8 (16 cost the long-context workload's followers a
// round trip on most long edges, 0.20 -> 0.27 ms); for leaders 16 was slower (1.9 -> 2.4 ms).
template <bool kLeader, int kFirst>
__device__ __forceinline__ void lane_walks(const TreeView* __restrict__ trees, int32_t p, const int32_t* req,
                                           int32_t len, int32_t known, bool act, int4 ce, int32_t& pos, int32_t& m,
                                           int4* ck, int32_t climit, int lane, int32_t* err) {
  while (__ballot_sync(kFull, act)) {
    int4 nn = make_int4(0, 0, 0, 0);
    int32_t k = 0, lim = 0, from2 = 0;
    const int32_t* lab = nullptr;
    bool need = false;
    if (act) {
      if (ce.w <= 0 || ce.y <= 0) {  // cannot happen in a valid tree
        atomicOr(err, ERR_CORRUPT_TREE);
        act = false;
      } else {
        nn = __ldg(trees[p].node + ce.y);
        lab = label_ptr(trees[p].label, trees[p].shared, ce.z);
        lim = min(ce.w, len - pos);
        const int32_t from = max(1, known - pos);
        k = lim;
        if (from < lim) {
          const int32_t first = min(lim, from + kFirst);
          k = first_diff_1(lab, req + pos, from, first);
          if (k == first && first < lim) {
            if (lim - first <= kThreadSpan) {
              k = first_diff_1(lab, req + pos, first, lim);
            } else {
              need = true;
              from2 = first;
            }
          }
        }
      }
    }
    for (unsigned needm = __ballot_sync(kFull, need); needm;) {
      const int j = __ffs(needm) - 1;
      const unsigned long long la = __shfl_sync(kFull, (unsigned long long)(uintptr_t)(lab + from2), j);
      const int32_t rp = __shfl_sync(kFull, pos + from2, j);
      const bool mine = need && (unsigned long long)(uintptr_t)(lab + from2) == la && pos + from2 == rp;
      const unsigned grp = __ballot_sync(kFull, mine);
      int32_t cmax = mine ? lim - from2 : 0;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) cmax = max(cmax, __shfl_xor_sync(kFull, cmax, o));
      const int32_t kk = compare_range<8, true>(reinterpret_cast<const int32_t*>(la), req + rp, 0, cmax, lane);
      if (mine) {
        k = from2 + min(kk < 0 ? cmax : kk, lim - from2);
        need = false;
      }
      needm &= ~grp;
    }
    if (act) {
      pos += k;
      m = pos;
      if (kLeader && ck && k == ce.w && pos <= climit) *ck = make_int4(pos, nn.x, nn.y, nn.z);
      act = k == ce.w && pos < len && nn.z > 0 &&
            find_child_1(trees[p].child + nn.x, tab_bits(nn.y), __ldg(req + pos), ce);
    }
  }
}

// The first two slots of the linear probe for tok in a table of 2^bits slots at tab (bits >= 2): 1 with
// e = the child, 0 if the child is absent, -1 if both slots hold other keys (the probe continues).
__device__ __forceinline__ int probe_first2(const int4& a, const int4& b, int32_t tok, int4& e) {
  if (a.y >= 1 && a.x == tok) {
    e = a;
    return 1;
  }
  if (a.y == 0) return 0;
  if (b.y >= 1 && b.x == tok) {
    e = b;
    return 1;
  }
  return b.y == 0 ? 0 : -1;
}

// One warp per request list[i], i < *count.
//   kLeader: the request is a group leader (or ungrouped): lane j walks trees j, j + 32, ..., and for a
//   leader with a checkpoint row records the checkpoints its followers resume from.
//   !kLeader: the request follows leader lead[f] with common prefix c = cpre[f]: match(f, T) = match(lead,
//   T) if that is < c, else a walk resumed at the leader's checkpoint that does not compare f's first c
//   tokens.  A lane takes kFollowIlp trees at a time (p, p + 32, ...): the leader's matches, the
//   checkpoints and the first probe step of each are loaded before any of them is looked at.
template <bool kLeader, bool kDecide, int kFirst = 8>
__global__ void __launch_bounds__(kFollowThreads, kFollowCtasPerSm) lane_kernel(
    const TreeView* __restrict__ trees, int32_t P, const int32_t* __restrict__ tokens, int64_t n_tokens,
    int64_t tok_base, const int64_t* __restrict__ offsets, const int32_t* __restrict__ list,
    const int32_t* __restrict__ count, const int32_t* __restrict__ lead, const int32_t* __restrict__ cpre,
    const int32_t* __restrict__ gid, const int32_t* __restrict__ cmin, int4* __restrict__ ckpt,
    const int32_t* __restrict__ load, int32_t alpha, int32_t* __restrict__ out_match, int32_t* __restrict__ out_peer,
    int32_t* err, int32_t* cursor, int32_t* __restrict__ out_next) {
  __shared__ unsigned long long s_top[kDecide ? kFollowThreads / 32 : 1][kDecide ? 64 : 1];
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kFollowThreads / 32);
  const int64_t n = *count;
  // Requests go to warps in a fixed stride, or, with a cursor (zero at launch), one at a time as warps
  // become free: leaders' walks differ widely in length.  The next index is fetched while the warp
  // routes the current request.
  int32_t nxt = 0;
  int64_t i0 = ((int64_t)blockIdx.x * kFollowThreads + threadIdx.x) >> 5;
  if (cursor) {
    if (lane == 0) nxt = atomicAdd(cursor, 1);
    i0 = __shfl_sync(kFull, nxt, 0);
  }
  for (int64_t i = i0; i < n; i = cursor ? (int64_t)__shfl_sync(kFull, nxt, 0) : i + warps) {
    if (cursor && lane == 0) nxt = atomicAdd(cursor, 1);
    const int64_t f = __ldg(list + i);
    const int64_t start = __ldg(offsets + f) - tok_base, end = __ldg(offsets + f + 1) - tok_base;
    const int64_t frow = f * P;
    if (!(start >= 0 && start <= end && end <= n_tokens)) {  // (followers are always valid)
      for (int32_t p = lane; p < P; p += 32) out_match[frow + p] = 0;
      if (lane == 0) {
        out_peer[f] = -1;
        if (kDecide && out_next) out_next[f] = -1;
        atomicOr(err, ERR_BAD_OFFSETS);
      }
      continue;
    }
    const int32_t* req = tokens + start;
    const int32_t len = (int32_t)min(end - start, (int64_t)INT32_MAX);
    LaneAcc<kDecide> acc(kDecide ? &s_top[threadIdx.x >> 5][lane] : nullptr);
    if constexpr (kLeader) {
      const int32_t row = __ldg(gid + f);
      const int32_t climit = row >= 0 ? __ldg(cmin + f) : -1;
      const int32_t tok0 = len > 0 ? __ldg(req) : 0;
      for (int32_t p0 = 0; p0 < P; p0 += 32) {
        const int32_t p = p0 + lane;
        int32_t m = 0, pos = 0;
        bool act = false;  // the lane has an edge to walk (ce, at position pos)
        int4 ce = make_int4(0, 0, 0, 0);
        int4* ck = nullptr;
        if (p < P && len > 0) {
          const int4 st = root_checkpoint(trees[p]);
          if (row >= 0) {
            ck = ckpt + (int64_t)row * P + p;
            *ck = st;
          }
          // The root filter answers most absent first tokens (fresh prompts) from L2; the root table only
          // when the token may be there.
          act = st.w > 0 && root_filter_has(trees[p].rfilter, tok0) &&
                find_child_1(trees[p].child + st.y, tab_bits(st.z), tok0, ce);
        }
        lane_walks<true, kFirst>(trees, p, req, len, 0, act, ce, pos, m, ck, climit, lane, err);
        if (p < P) {
          out_match[frow + p] = m;
          acc.add(m, __ldg(load + p), p, alpha);
        }
      }
    } else {
      const int32_t c = __ldg(cpre + f);
      const int32_t l = __ldg(lead + f);
      const int32_t row = __ldg(gid + l);
      const int64_t lrow = (int64_t)l * P;  // the leaders' pass has finished: the leader's row is final
      const int4* ckrow = ckpt + (int64_t)(row >= 0 ? row : 0) * P;
      for (int32_t p0 = 0; p0 < P; p0 += 32 * kFollowIlp) {
        int32_t pt[kFollowIlp], ml[kFollowIlp], pos[kFollowIlp], m[kFollowIlp], tk[kFollowIlp];
        bool act[kFollowIlp];
        int4 st[kFollowIlp], e0[kFollowIlp], e1[kFollowIlp], ce[kFollowIlp];
        const int4* tab[kFollowIlp];
#pragma unroll
        for (int g = 0; g < kFollowIlp; ++g) {
          pt[g] = p0 + 32 * g + lane;
          ml[g] = pt[g] < P ? out_match[lrow + pt[g]] : 0;
          // The checkpoint is loaded with the leader's match, before the match says whether it is needed:
          // a group's followers are routed side by side, so its row is in cache, and one round trip is saved.
          st[g] = pt[g] < P && row >= 0 ? ckrow[pt[g]] : make_int4(0, 0, 0, 0);
        }
#pragma unroll
        for (int g = 0; g < kFollowIlp; ++g) {
          const bool w = pt[g] < P && len > 0 && ml[g] >= c && c < len;
          if (!w) st[g] = make_int4(0, 0, 0, 0);
          else if (row < 0) st[g] = root_checkpoint(trees[pt[g]]);
          pos[g] = min(st[g].x, len);
          m[g] = w ? pos[g] : len == 0 ? 0 : ml[g] < c ? ml[g] : len;
          act[g] = w && pos[g] < len && st[g].w > 0 && tab_bits(st[g].z) > 0;
        }
#pragma unroll
        for (int g = 0; g < kFollowIlp; ++g) tk[g] = act[g] ? __ldg(req + pos[g]) : 0;
#pragma unroll
        for (int g = 0; g < kFollowIlp; ++g) {
          e0[g] = e1[g] = ce[g] = make_int4(0, 0, 0, 0);
          tab[g] = nullptr;
          if (act[g]) {
            const int32_t bits = tab_bits(st[g].z);
            const uint32_t mask = (1u << bits) - 1, h = slot_hash(tk[g], bits);
            tab[g] = trees[pt[g]].child + st[g].y;
            e0[g] = __ldg(tab[g] + h);
            e1[g] = __ldg(tab[g] + ((h + 1) & mask));
          }
        }
#pragma unroll
        for (int g = 0; g < kFollowIlp; ++g) {
          if (act[g]) {
            const int r = probe_first2(e0[g], e1[g], tk[g], ce[g]);
            act[g] = r > 0 || (r < 0 && find_child_1(tab[g], tab_bits(st[g].z), tk[g], ce[g]));
          }
        }
#pragma unroll
        for (int g = 0; g < kFollowIlp; ++g) {
          lane_walks<false, kFirst>(trees, pt[g], req, len, c, act[g], ce[g], pos[g], m[g], nullptr, -1, lane, err);
          if (pt[g] < P) {
            out_match[frow + pt[g]] = m[g];
            acc.add(m[g], __ldg(load + pt[g]), pt[g], alpha);
          }
        }
      }
    }
    acc.finish(lane, f, out_peer, out_next);
  }
}

// Route decision from a match matrix with excluded peers: the best and the next-best candidate by the route
// order of route_key, skipping trees whose staged load word carries kExcluded (Section 3.2: a peer that
// pushes back; Section 3.3: a suspected-failed peer, and the next-best target a request falls back to when
// forwarding times out).  Match values below 0 count as 0.
//
// Up to 256 trees (P a multiple of 4, the matrix on a 16-byte boundary) a row is read by 8 lanes, four rows
// per warp at a time: lane j of a row's group takes columns 32i + 4j .. 32i + 4j + 3 (i < 8, one 16-byte load
// each), so a group reads 128 contiguous bytes per load.  The route order of a column is its score
// m - alpha * load, then its tie-break (lower load, then lower index), which is a fixed order of the columns:
// with rank(p) = the number of columns p comes before on the tie-break, a unique 8-bit value, the order is
// that of the 32-bit key (m - alpha * load + 2^22) * 256 + rank(p) whenever 0 <= m < 2^22 and
// 0 <= alpha * load < 2^22 (the key then lies in [256, 2^31)).  A lane holds (2^22 - alpha * load) * 256 + rank
// of each of its columns (INT_MIN for an excluded one, so its key stays negative), and a column costs one
// shift-add and three min/max for the top two keys.  A warp's four rows take the 64-bit keys of RouteAcc
// instead when one of their values is outside [0, 2^22), and every row does when a load term is 2^22 or more.
// Other shapes take one warp per row with RouteAcc<true>.
constexpr int kDecideUnroll = 8;        // columns a lane loads per stretch on the one-warp-per-row path
constexpr int32_t kSmallKey = 1 << 22;  // bound on match values and load terms of the 32-bit keys
__global__ void __launch_bounds__(256, 2) decide_kernel(const int32_t* __restrict__ match, int64_t B, int32_t P,
                                                     const int32_t* __restrict__ load, int32_t alpha,
                                                     int32_t* __restrict__ out_peer, int32_t* __restrict__ out_next) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  if (P <= 256 && P % 4 == 0 && (reinterpret_cast<uintptr_t>(match) & 15) == 0) {
    __shared__ int32_t s_rank[256];   // tie-break rank of each column
    __shared__ int16_t s_col[256];    // the column of each rank
    for (int32_t p = threadIdx.x; p < P; p += blockDim.x) {
      const int32_t lp = __ldg(load + p) & 0xFFFF;
      int32_t r = 0;
      for (int32_t q = 0; q < P; ++q) {
        const int32_t lq = __ldg(load + q) & 0xFFFF;
        r += lq > lp || (lq == lp && q > p);
      }
      s_rank[p] = r;
      s_col[r] = (int16_t)p;
    }
    __syncthreads();
    const int j = lane & 7;
    int32_t base[32];
    bool small = true;
#pragma unroll
    for (int c = 0; c < 32; ++c) {
      const int32_t p = 32 * (c >> 2) + 4 * j + (c & 3);
      base[c] = INT_MIN;
      if (p < P) {
        const int32_t ldw = __ldg(load + p);
        const long long term = (long long)alpha * (ldw & 0xFFFF);
        if (!(ldw & kExcluded)) {
          if (term < kSmallKey)
            base[c] = (int32_t)(((kSmallKey - term) << 8) | s_rank[p]);
          else
            small = false;
        }
      }
    }
    small = __all_sync(kFull, small);  // every warp holds every column, so every warp agrees
    const int64_t quads = (B + 3) / 4;
    for (int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; w < quads; w += warps) {
      const int64_t b = 4 * w + (lane >> 3);
      const bool row_ok = b < B;
      const int4* r4 = reinterpret_cast<const int4*>(match + (row_ok ? b : 0) * P + 4 * j);
      int4 v[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = row_ok && 32 * i + 4 * j < P ? __ldg(r4 + 8 * i) : make_int4(0, 0, 0, 0);
      uint32_t any = 0;  // OR of the values: below 2^22 (unsigned) iff every value is in [0, 2^22)
#pragma unroll
      for (int i = 0; i < 8; ++i) any |= (uint32_t)(v[i].x | v[i].y | v[i].z | v[i].w);
      if (small && !__any_sync(kFull, any >= (uint32_t)kSmallKey)) {
        int32_t k1 = 0, k2 = 0;
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          const int4& x = v[c >> 2];
          const int32_t m = (c & 3) == 0 ? x.x : (c & 3) == 1 ? x.y : (c & 3) == 2 ? x.z : x.w;
          const int32_t key = (m << 8) + base[c];
          k2 = max(k2, min(k1, key));
          k1 = max(k1, key);
        }
#pragma unroll
        for (int o = 4; o > 0; o >>= 1) {
          const int32_t o1 = __shfl_xor_sync(kFull, k1, o), o2 = __shfl_xor_sync(kFull, k2, o);
          k2 = max(min(k1, o1), max(k2, o2));
          k1 = max(k1, o1);
        }
        if (j == 0 && row_ok) {
          out_peer[b] = k1 > 0 ? s_col[k1 & 0xFF] : -1;
          if (out_next) out_next[b] = k2 > 0 ? s_col[k2 & 0xFF] : -1;
        }
      } else {
        RouteAcc<true> acc;
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          const int32_t p = 32 * (c >> 2) + 4 * j + (c & 3);
          const int4& x = v[c >> 2];
          const int32_t m = (c & 3) == 0 ? x.x : (c & 3) == 1 ? x.y : (c & 3) == 2 ? x.z : x.w;
          if (p < P) acc.add(max(m, 0), __ldg(load + p), p, alpha);
        }
        acc.warp_merge(4);
        if (j == 0 && row_ok) acc.write(b, out_peer, out_next);
      }
    }
    return;
  }
  for (int64_t b = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; b < B; b += warps) {
    const int32_t* row = match + b * P;
    RouteAcc<true> acc;
    for (int32_t p0 = 0; p0 < P; p0 += 32 * kDecideUnroll) {
      int32_t v[kDecideUnroll];  // a lane's columns of this stretch, loaded before any is looked at
#pragma unroll
      for (int u = 0; u < kDecideUnroll; ++u) {
        const int32_t p = p0 + 32 * u + lane;
        v[u] = p < P ? __ldg(row + p) : 0;
      }
#pragma unroll
      for (int u = 0; u < kDecideUnroll; ++u) {
        const int32_t p = p0 + 32 * u + lane;
        if (p < P) acc.add(max(v[u], 0), __ldg(load + p), p, alpha);
      }
    }
    acc.warp_merge();
    if (lane == 0) acc.write(b, out_peer, out_next);
  }
}

}  // namespace

namespace {

// The leader and follower passes with the decision of RouteAcc<kDecide>.
template <bool kDecide>
cudaError_t launch_passes(const TreeView* d_trees, int32_t P, const int32_t* tokens, int64_t n_tokens, int64_t tok_base,
                          const int64_t* offsets, int64_t B, const int32_t* d_load, int32_t alpha, int32_t* out_match,
                          int32_t* out_peer, int32_t* d_err, const GroupScratch* g, int num_sms, cudaStream_t st,
                          int32_t* out_next, int* launched) {
  const int64_t want = (B + kFollowThreads / 32 - 1) / (kFollowThreads / 32);
  const int grid2 = (int)std::min<int64_t>(want, (int64_t)num_sms * kFollowCtasPerSm);
  cudaError_t e;
  if (n_tokens >= B * (int64_t)kSlotTokens) {
    // Requests of a staging window or longer on average: the leaders' walks are long compares, which the
    // staged kernel's warps do from shared memory.
    const size_t smem = (size_t)kSlots * kSlotTokens * sizeof(int32_t);
    e = cudaFuncSetAttribute(route_kernel<kDecide>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int64_t max_ctas = (int64_t)num_sms * kCtasPerSm;
    const int grid = (int)(B < max_ctas ? B : max_ctas);
    P2P_TIMED(K_ROUTE_STAGED, st,
              (route_kernel<kDecide><<<grid, kThreads, smem, st>>>(d_trees, P, tokens, n_tokens, tok_base, offsets, B,
                                                                   g->lists, g->counts, g->gid, g->cmin, g->ckpt, d_load,
                                                                   alpha, out_match, out_peer, d_err, out_next)));
    *launched = 1;
  } else {
    // Shorter requests: most leader walks end within a few tokens, so each lane walks its own tree.
    P2P_TIMED(K_LANE_LEADER, st,
              (lane_kernel<true, kDecide><<<grid2, kFollowThreads, 0, st>>>(
                  d_trees, P, tokens, n_tokens, tok_base, offsets, g->lists, g->counts, nullptr, nullptr, g->gid,
                  g->cmin, g->ckpt, d_load, alpha, out_match, out_peer, d_err, g->counts + 3, out_next)));
    *launched = 1;
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // The followers' first per-lane compare: 8 tokens for long requests, 16 otherwise (lane_walks).
  if (n_tokens >= B * (int64_t)kSlotTokens) {
    P2P_TIMED(K_LANE_FOLLOWER, st,
              (lane_kernel<false, kDecide, 8><<<grid2, kFollowThreads, 0, st>>>(
                  d_trees, P, tokens, n_tokens, tok_base, offsets, g->lists + B, g->counts + 1, g->lead, g->cpre, g->gid,
                  nullptr, g->ckpt, d_load, alpha, out_match, out_peer, d_err, nullptr, out_next)));
  } else {
    P2P_TIMED(K_LANE_FOLLOWER, st,
              (lane_kernel<false, kDecide, 16><<<grid2, kFollowThreads, 0, st>>>(
                  d_trees, P, tokens, n_tokens, tok_base, offsets, g->lists + B, g->counts + 1, g->lead, g->cpre, g->gid,
                  nullptr, g->ckpt, d_load, alpha, out_match, out_peer, d_err, nullptr, out_next)));
  }
  *launched += 1;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_route(const TreeView* d_trees, int32_t P, const int32_t* tokens, int64_t n_tokens, int64_t tok_base,
                         const int64_t* offsets, int64_t B, const int32_t* d_load, int32_t alpha, int32_t* out_match,
                         int32_t* out_peer, int32_t* d_err, const GroupScratch* g, int num_sms, cudaStream_t st,
                         int* launched, bool decide, int32_t* out_next) {
  *launched = 0;
  if (B <= 0) return cudaSuccess;
  if (!g) return cudaErrorInvalidValue;  // every batch is grouped first
  if (decide || out_next)
    return launch_passes<true>(d_trees, P, tokens, n_tokens, tok_base, offsets, B, d_load, alpha, out_match, out_peer,
                               d_err, g, num_sms, st, out_next, launched);
  return launch_passes<false>(d_trees, P, tokens, n_tokens, tok_base, offsets, B, d_load, alpha, out_match, out_peer,
                              d_err, g, num_sms, st, nullptr, launched);
}

cudaError_t launch_decide(const int32_t* match, int64_t B, int32_t P, const int32_t* d_load, int32_t alpha,
                          int32_t* out_peer, int32_t* out_next, int num_sms, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  // One wave of resident CTAs (the kernel's registers allow 2 per SM): every CTA ranks the columns once.
  const int64_t want = (B + 7) / 8;
  const int grid = (int)std::min<int64_t>(want, (int64_t)std::max(num_sms, 1) * 2);
  P2P_TIMED(K_DECIDE, st, (decide_kernel<<<grid, 256, 0, st>>>(match, B, P, d_load, alpha, out_peer, out_next)));
  return cudaGetLastError();
}

}  // namespace p2p
