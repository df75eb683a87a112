// group_kernel.cu -- shared-prefix groups of a request batch, ahead of the route kernel.
//
// Requests of one batch often share long prefixes (a few-shot or system prompt in front of each query).
// Their walks in a tree coincide along the shared part, so a batch is routed in two passes: group leaders
// walk every tree as usual, and every other request of a group (a follower) starts from its leader's result.
// For a follower f of leader l with c = LCP(r_f, r_l) (exact, computed here):
//   - if match(r_l, T) < c, then match(r_f, T) = match(r_l, T): both walks stop at the same token;
//   - otherwise match(r_f, T) >= c, and the follower's walk need not compare its first c tokens.
// Both facts hold for the PrefixMatch of Algorithm 1 because a walk depends only on the request tokens it
// has consumed.  Results are therefore identical to independent walks; grouping changes only the work.
//
// Grouping: a request of at least kGroupHead tokens is keyed by a 64-bit hash of its first kGroupHead tokens
// and inserted into an open-addressing table; the smallest request index with that key leads the group.
// A follower whose exact common prefix with its leader is shorter than kGroupHead (a hash collision) routes
// as a leader instead.  The leader choice is deterministic (smallest index); the order of the two request
// lists is not, and only affects scheduling.  Each group's followers take a contiguous range of the follower
// list (group_ranges_kernel, group_place_kernel): the warps that route them at the same time then read the
// leader's match row, its checkpoints and the tables at the checkpoint nodes once, from cache.
#include "internal.h"

namespace p2p {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kGroupThreads = 256;

// SplitMix64 output function (Steele, Lea & Flood 2014; constants published by Vigna).
__device__ __forceinline__ unsigned long long mix64(unsigned long long z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ bool request_range(const int64_t* offsets, int64_t b, int64_t tok_base, int64_t n_tokens,
                                              int64_t& start, int64_t& len) {
  start = offsets[b] - tok_base;
  const int64_t end = offsets[b + 1] - tok_base;
  len = end - start;
  return start >= 0 && start <= end && end <= n_tokens;
}

// One warp per 32 consecutive requests (lane i owns request base + i).  The warp hashes each request's
// first kGroupHead tokens in turn (one token per lane and position, each mixed with its position, summed);
// then every distinct key of the 32 is looked up or claimed once, by its lowest lane, which also lowers
// the key's leader index to that lane's request (the smallest of the warp's requests with the key).
__global__ void __launch_bounds__(kGroupThreads) group_hash_kernel(
    const int32_t* __restrict__ tokens, int64_t n_tokens, int64_t tok_base, const int64_t* __restrict__ offsets,
    int64_t B, unsigned long long* keys, int32_t* vals, int32_t bits, int32_t* slot_of) {
  static_assert(kGroupHead == 64, "two tokens per lane");
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kGroupThreads / 32);
  const uint32_t mask = (1u << bits) - 1;
  for (int64_t base = (((int64_t)blockIdx.x * kGroupThreads + threadIdx.x) >> 5) * 32; base < B; base += warps * 32) {
    unsigned long long my_h = 0;  // 0: the lane's request is not grouped
    for (int r = 0; r < 32 && base + r < B; ++r) {
      int64_t start, len;
      if (!request_range(offsets, base + r, tok_base, n_tokens, start, len) || len < kGroupHead) continue;
      const int32_t* g = tokens + start;
      unsigned long long h = mix64((unsigned long long)(uint32_t)__ldg(g + lane) | ((unsigned long long)lane << 32)) +
                             mix64((unsigned long long)(uint32_t)__ldg(g + lane + 32) |
                                   ((unsigned long long)(lane + 32) << 32));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) h += __shfl_xor_sync(kFull, h, o);
      h |= 1ull;  // 0 marks an empty slot
      if (lane == r) my_h = h;
    }
    const unsigned same = __match_any_sync(kFull, my_h);
    const int first = __ffs(same) - 1;
    int32_t slot = -1;
    if (my_h && lane == first) {
      uint32_t sl = (uint32_t)my_h & mask;
      for (uint32_t it = 0; it <= mask; ++it, sl = (sl + 1) & mask) {
        const unsigned long long prev = atomicCAS(&keys[sl], 0ull, my_h);
        if (prev == 0ull || prev == my_h) {
          slot = (int32_t)sl;
          break;
        }
      }
      if (slot >= 0) atomicMin(&vals[slot], (int32_t)(base + lane));
    }
    slot = __shfl_sync(kFull, slot, first);
    if (base + lane < B) slot_of[base + lane] = my_h ? slot : -1;
  }
}

// First position in [0, n) where a and b differ, or n (one warp, both in global memory).
__device__ int64_t lcp_warp(const int32_t* __restrict__ a, const int32_t* __restrict__ b, int64_t n, int lane) {
  constexpr int U = 8;
  int64_t j0 = 0;
  for (; j0 + 32 * U <= n; j0 += 32 * U) {
    int32_t x[U];
#pragma unroll
    for (int u = 0; u < U; ++u) x[u] = __ldg(a + j0 + u * 32 + lane);
    int32_t diff = 0;
#pragma unroll
    for (int u = 0; u < U; ++u) diff |= x[u] ^ __ldg(b + j0 + u * 32 + lane);
    if (__any_sync(kFull, diff != 0)) {
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const unsigned m = __ballot_sync(kFull, x[u] != __ldg(b + j0 + u * 32 + lane));
        if (m) return j0 + u * 32 + (__ffs(m) - 1);
      }
    }
  }
  for (; j0 < n; j0 += 32) {
    const int64_t j = j0 + lane;
    const unsigned m = __ballot_sync(kFull, j < n && __ldg(a + j) != __ldg(b + j));
    if (m) return j0 + (__ffs(m) - 1);
  }
  return n;
}

// One warp per 32 consecutive requests (lane i owns request base + i): each request's leader; for each
// follower in turn, the exact common prefix with its leader (the whole warp compares); then the warp's
// leaders are appended to lists[0 ..) with one counter update, and each follower takes its rank in its group
// (fcnt[leader] counts them; the rank goes to slot_of[b]).  counts and fcnt must start at zero, gid at -1 and
// cmin at INT32_MAX.  A leader with followers gets the smallest of their common prefixes in cmin and, while
// rows last, a checkpoint row in gid (one update per distinct leader of the warp's followers).
__global__ void __launch_bounds__(kGroupThreads) group_resolve32_kernel(
    const int32_t* __restrict__ tokens, int64_t n_tokens, int64_t tok_base, const int64_t* __restrict__ offsets,
    int64_t B, const int32_t* __restrict__ vals, int32_t* slot_of, int32_t* lead, int32_t* cpre, int32_t* lists,
    int32_t* counts, int32_t* gid, int32_t* cmin, int32_t gcap, int32_t* fcnt) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kGroupThreads / 32);
  for (int64_t base = (((int64_t)blockIdx.x * kGroupThreads + threadIdx.x) >> 5) * 32; base < B; base += warps * 32) {
    const int64_t b = base + lane;
    const bool valid = b < B;
    const int32_t s = valid ? slot_of[b] : -1;
    const int32_t l = s >= 0 ? vals[s] : (int32_t)b;
    int32_t my_c = -1;
    for (unsigned fm = __ballot_sync(kFull, valid && l != (int32_t)b); fm; fm &= fm - 1) {
      const int r = __ffs(fm) - 1;
      const int32_t lr = __shfl_sync(kFull, l, r);
      int64_t sb, nb, sl, nl;  // both requests are valid and hold at least kGroupHead tokens
      request_range(offsets, base + r, tok_base, n_tokens, sb, nb);
      request_range(offsets, lr, tok_base, n_tokens, sl, nl);
      int64_t c = lcp_warp(tokens + sb, tokens + sl, min(nb, nl), lane);
      if (c < kGroupHead || c > INT32_MAX) c = -1;
      if (lane == r) my_c = (int32_t)c;
    }
    const bool is_f = my_c >= 0;
    const unsigned lm = __ballot_sync(kFull, valid && !is_f), fm = __ballot_sync(kFull, is_f);
    int32_t lbase = 0, fbase = 0;
    if (lane == 0) {
      if (lm) lbase = atomicAdd(&counts[0], __popc(lm));
      if (fm) fbase = atomicAdd(&counts[1], __popc(fm));
    }
    lbase = __shfl_sync(kFull, lbase, 0);
    fbase = __shfl_sync(kFull, fbase, 0);
    const unsigned below = (1u << lane) - 1;
    if (valid && !is_f) {
      lead[b] = (int32_t)b;
      lists[lbase + __popc(lm & below)] = (int32_t)b;
    }
    (void)fbase;
    const unsigned same = __match_any_sync(kFull, is_f ? l : -1);
    if (is_f) {
      lead[b] = l;
      cpre[b] = my_c;
      const int32_t c_min = (int32_t)__reduce_min_sync(same, (unsigned)my_c);
      const int first = __ffs(same) - 1;
      int32_t rbase = 0;
      if (lane == first) {
        atomicMin(&cmin[l], c_min);
        rbase = atomicAdd(&fcnt[l], __popc(same));
        if (atomicCAS(&gid[l], -1, -2) == -1) {  // the leader's first follower gives it a row
          const int32_t row = atomicAdd(&counts[2], 1);
          atomicExch(&gid[l], row < gcap ? row : -1);
        }
      }
      slot_of[b] = __shfl_sync(same, rbase, first) + __popc(same & below);  // rank in the group
    }
  }
}

// One warp per request: its leader and the exact common prefix with it; the CTA's leaders of a round are
// then appended to lists[0 ..) with one counter update per round, and the followers counted (one update per
// round) and ranked in their groups as in group_resolve32_kernel.  counts and fcnt must start at zero, gid at
// -1 and cmin at INT32_MAX.  A leader with followers gets the smallest of their common prefixes in cmin
// (updated only when a follower lowers it, so popular groups make few atomics) and, while rows last, a
// checkpoint row in gid.
__global__ void __launch_bounds__(kGroupThreads) group_resolve_kernel(
    const int32_t* __restrict__ tokens, int64_t n_tokens, int64_t tok_base, const int64_t* __restrict__ offsets,
    int64_t B, const int32_t* __restrict__ vals, int32_t* slot_of, int32_t* lead, int32_t* cpre, int32_t* lists,
    int32_t* counts, int32_t* gid, int32_t* cmin, int32_t gcap, int32_t* fcnt) {
  constexpr int kWarps = kGroupThreads / 32;
  __shared__ int s_kind[kWarps];  // 0: none, 1: leader, 2: follower
  __shared__ int s_pos[kWarps];   // the request's index in its list
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int64_t r0 = (int64_t)blockIdx.x * kWarps; r0 < B; r0 += (int64_t)gridDim.x * kWarps) {
    const int64_t b = r0 + warp;
    int kind = 0;
    int32_t l = -1, c32 = -1;
    if (b < B) {
      const int32_t s = slot_of[b];
      l = s >= 0 ? vals[s] : (int32_t)b;
      int64_t c = -1;
      if (l != (int32_t)b) {  // both requests are valid and hold at least kGroupHead tokens
        int64_t sb, nb, sl, nl;
        request_range(offsets, b, tok_base, n_tokens, sb, nb);
        request_range(offsets, l, tok_base, n_tokens, sl, nl);
        c = lcp_warp(tokens + sb, tokens + sl, min(nb, nl), lane);
        if (c < kGroupHead || c > INT32_MAX) c = -1;
      }
      kind = c < 0 ? 1 : 2;
      c32 = (int32_t)c;
    }
    if (lane == 0) s_kind[warp] = kind;
    __syncthreads();
    if (threadIdx.x == 0) {
      int nl = 0, nf = 0;
      for (int w = 0; w < kWarps; ++w) nl += s_kind[w] == 1, nf += s_kind[w] == 2;
      const int bl = nl ? atomicAdd(&counts[0], nl) : 0, bf = nf ? atomicAdd(&counts[1], nf) : 0;
      for (int w = 0, il = 0, jf = 0; w < kWarps; ++w) s_pos[w] = s_kind[w] == 1 ? bl + il++ : s_kind[w] == 2 ? bf + jf++ : 0;
    }
    __syncthreads();
    if (lane == 0 && kind == 1) {
      lead[b] = (int32_t)b;
      lists[s_pos[warp]] = (int32_t)b;
    } else if (lane == 0 && kind == 2) {
      lead[b] = l;
      cpre[b] = c32;
      slot_of[b] = atomicAdd(&fcnt[l], 1);  // rank in the group (slot_of[b] was read above)
      if (c32 < *(volatile int32_t*)&cmin[l]) atomicMin(&cmin[l], c32);
      if (*(volatile int32_t*)&gid[l] == -1 && atomicCAS(&gid[l], -1, -2) == -1) {
        const int32_t row = atomicAdd(&counts[2], 1);  // the leader's first follower gives it a row
        atomicExch(&gid[l], row < gcap ? row : -1);
      }
    }
    __syncthreads();  // s_kind and s_pos are reused next round
  }
}

// Gives every leader with followers a contiguous range of the follower list: fcnt[l] (its follower count)
// becomes the start of the range.  One warp per 32 consecutive requests: an inclusive scan of their counts
// and one counter update per warp (counts[4]).
__global__ void __launch_bounds__(kGroupThreads) group_ranges_kernel(int64_t B, int32_t* fcnt, int32_t* counts) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kGroupThreads / 32);
  for (int64_t base = (((int64_t)blockIdx.x * kGroupThreads + threadIdx.x) >> 5) * 32; base < B; base += warps * 32) {
    const int64_t b = base + lane;
    const int32_t c = b < B ? fcnt[b] : 0;  // zero for every request that leads no follower
    int32_t incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t v = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += v;
    }
    int32_t off = 0;
    if (lane == 31 && incl) off = atomicAdd(&counts[4], incl);
    off = __shfl_sync(kFull, off, 31);
    if (c) fcnt[b] = off + incl - c;
  }
}

// Places follower b at lists[B + start of its leader's range + its rank in the group].
__global__ void __launch_bounds__(kGroupThreads) group_place_kernel(int64_t B, const int32_t* __restrict__ lead,
                                                                    const int32_t* __restrict__ rank,
                                                                    const int32_t* __restrict__ fcnt, int32_t* lists) {
  const int64_t stride = (int64_t)gridDim.x * kGroupThreads;
  for (int64_t b = (int64_t)blockIdx.x * kGroupThreads + threadIdx.x; b < B; b += stride) {
    const int32_t l = lead[b];
    if (l != (int32_t)b) lists[B + fcnt[l] + rank[b]] = (int32_t)b;
  }
}

}  // namespace

cudaError_t launch_group(const int32_t* tokens, int64_t n_tokens, int64_t tok_base, const int64_t* offsets, int64_t B,
                         const GroupScratch& g, int num_sms, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  const size_t slots = (size_t)1 << g.bits;
  cudaError_t e = cudaMemsetAsync(g.keys, 0, slots * sizeof(unsigned long long), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(g.vals, 0x7f, slots * sizeof(int32_t), st);  // 0x7f7f7f7f > any index
  if (e == cudaSuccess) e = cudaMemsetAsync(g.counts, 0, 8 * sizeof(int32_t), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(g.fcnt, 0, (size_t)B * sizeof(int32_t), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(g.gid, 0xff, (size_t)B * sizeof(int32_t), st);   // -1
  if (e == cudaSuccess) e = cudaMemsetAsync(g.cmin, 0x7f, (size_t)B * sizeof(int32_t), st);  // > any prefix
  if (e != cudaSuccess) return e;
  const int64_t hash_ctas = ((B + 31) / 32 + kGroupThreads / 32 - 1) / (kGroupThreads / 32);  // a warp per 32 requests
  const int64_t resolve_ctas = (B + kGroupThreads / 32 - 1) / (kGroupThreads / 32);            // a warp per request
  const int grid = (int)std::min<int64_t>(hash_ctas, (int64_t)num_sms * 8);
  const int grid2 = (int)std::min<int64_t>(resolve_ctas, (int64_t)num_sms * 8);
  P2P_TIMED(K_GROUP_HASH, st,
            (group_hash_kernel<<<grid, kGroupThreads, 0, st>>>(tokens, n_tokens, tok_base, offsets, B, g.keys, g.vals,
                                                               g.bits, g.slot_of)));
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // Large batches: a warp per 32 requests (at least 32 warps per SM still busy; fewest atomics).  Smaller
  // ones: a warp per request, so that the common-prefix compares spread over as many warps as there are
  // requests.
  if (B >= (int64_t)num_sms * 32 * 32) {
    P2P_TIMED(K_GROUP_RESOLVE32, st,
              (group_resolve32_kernel<<<grid, kGroupThreads, 0, st>>>(tokens, n_tokens, tok_base, offsets, B, g.vals,
                                                                      g.slot_of, g.lead, g.cpre, g.lists, g.counts,
                                                                      g.gid, g.cmin, g.gcap, g.fcnt)));
  } else {
    P2P_TIMED(K_GROUP_RESOLVE, st,
              (group_resolve_kernel<<<grid2, kGroupThreads, 0, st>>>(tokens, n_tokens, tok_base, offsets, B, g.vals,
                                                                     g.slot_of, g.lead, g.cpre, g.lists, g.counts,
                                                                     g.gid, g.cmin, g.gcap, g.fcnt)));
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // Each group's followers side by side in the follower list.
  const int64_t place_ctas = (B + kGroupThreads - 1) / kGroupThreads;
  const int grid3 = (int)std::min<int64_t>(place_ctas, (int64_t)num_sms * 8);
  P2P_TIMED(K_GROUP_RANGES, st, (group_ranges_kernel<<<grid, kGroupThreads, 0, st>>>(B, g.fcnt, g.counts)));
  P2P_TIMED(K_GROUP_PLACE, st,
            (group_place_kernel<<<grid3, kGroupThreads, 0, st>>>(B, g.lead, g.slot_of, g.fcnt, g.lists)));
  return cudaGetLastError();
}

}  // namespace p2p
