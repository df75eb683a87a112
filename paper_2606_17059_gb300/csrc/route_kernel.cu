// route_kernel.cu -- batched longest-prefix match against P radix trees and the route decision.
//
// Computes, for every request r_b and tree T_p, match(r_b, T_p) = PrefixMatch of Algorithm 1 (the
// number of leading request tokens found along one path of T_p, a partial edge included), and the
// chosen peer argmax_p (match - alpha*load_p, -load_p, -p) (Algorithm 1's argmax with a load term).
//
// Mapping: one CTA owns one request at a time (grid-stride over requests).  The request's tokens are
// staged once into shared memory and shared by the CTA's warps; warp w walks trees w, w+W, ...  A walk
// is warp-cooperative: a child lookup probes 32 slots of the node's children hash table at once (one
// coalesced load, whatever the fan-out), and an edge label is compared 32 tokens per load with several
// loads in flight per lane; the first mismatch comes from __ballot_sync + __ffs.  Each warp keeps the best packed route
// key of its trees; the CTA reduces the W keys in shared memory.  Integer work only: no tensor cores.
#include "internal.h"

namespace p2p {
namespace {

constexpr int kWarps = 8;                 // warps per CTA
constexpr int kThreads = kWarps * 32;
constexpr int kUnroll = 4;                // label loads in flight per lane (128 tokens per warp step)
constexpr int kSmemTokens = 4096;         // request tokens staged in shared memory (16 KB)
constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ int32_t req_at(const int32_t* s_req, int32_t n_s, const int32_t* g_req, int64_t i) {
  return i < n_s ? s_req[i] : __ldg(g_req + i);
}

// Child with first token `tok` in the children table of 2^bits slots at tab: one coalesced probe of 32
// consecutive slots (a table is at most 3/4 full, so the probe run almost always fits).  Returns false if
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

// First j in [1, lim) with lab[j] != request[pos + j], or lim.  lab[0] == request[pos] is known.
__device__ __forceinline__ int64_t first_mismatch(const int32_t* __restrict__ lab, const int32_t* s_req, int32_t n_s,
                                                  const int32_t* g_req, int64_t pos, int64_t lim, int lane) {
  for (int64_t j0 = 1; j0 < lim; j0 += kUnroll * 32) {
    int32_t v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t j = j0 + u * 32 + lane;
      v[u] = j < lim ? __ldg(lab + j) : 0;
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t j = j0 + u * 32 + lane;
      const bool ne = j < lim && v[u] != req_at(s_req, n_s, g_req, pos + j);
      const unsigned m = __ballot_sync(kFull, ne);
      if (m) return j0 + u * 32 + (__ffs(m) - 1);
    }
  }
  return lim;
}

// match(r, T) for one tree, computed by the whole warp (result uniform across lanes).
__device__ int32_t walk(const TreeView& t, const int32_t* s_req, int32_t n_s, const int32_t* g_req, int64_t len,
                        int lane, int32_t* err) {
  if (len == 0) return 0;
  int4 ce;
  if (!find_child(t.child + t.root_off, t.root_bits, req_at(s_req, n_s, g_req, 0), lane, ce)) return 0;
  int64_t pos = 0;
  for (;;) {
    if (ce.w <= 0 || ce.y <= 0) {  // cannot happen in a valid tree; keeps the loop finite if it does
      if (lane == 0) atomicOr(err, ERR_CORRUPT_TREE);
      break;
    }
    const int4 nn = __ldg(t.node + ce.y);  // the child's record, fetched while its label is compared
    const int64_t lim = min((int64_t)ce.w, len - pos);
    const int64_t k = first_mismatch(t.label + ce.z, s_req, n_s, g_req, pos, lim, lane);
    pos += k;
    if (k < ce.w || pos >= len || nn.z <= 0) break;
    if (!find_child(t.child + nn.x, tab_bits(nn.y), req_at(s_req, n_s, g_req, pos), lane, ce)) break;
  }
  return (int32_t)pos;
}

__global__ void __launch_bounds__(kThreads) route_kernel(const TreeView* __restrict__ trees, int32_t P,
                                                         const int32_t* __restrict__ tokens, int64_t n_tokens,
                                                         int64_t tok_base, const int64_t* __restrict__ offsets,
                                                         int64_t B, const int32_t* __restrict__ load, int32_t alpha,
                                                         int32_t* __restrict__ out_match,
                                                         int32_t* __restrict__ out_peer, int32_t* err) {
  extern __shared__ int32_t s_req[];
  __shared__ unsigned long long s_best[kWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int64_t b = blockIdx.x; b < B; b += gridDim.x) {
    const int64_t start = __ldg(offsets + b) - tok_base, end = __ldg(offsets + b + 1) - tok_base;
    if (!(start >= 0 && start <= end && end <= n_tokens)) {  // same for every thread of the CTA
      for (int32_t p = threadIdx.x; p < P; p += kThreads) out_match[b * P + p] = 0;
      if (threadIdx.x == 0) {
        out_peer[b] = -1;
        atomicOr(err, ERR_BAD_OFFSETS);
      }
      continue;
    }
    const int64_t len = end - start;
    const int32_t* g_req = tokens + start;
    const int32_t n_s = (int32_t)min(len, (int64_t)kSmemTokens);
    for (int32_t i = threadIdx.x; i < n_s; i += kThreads) s_req[i] = __ldg(g_req + i);
    __syncthreads();
    unsigned long long best = 0;
    for (int32_t p = warp; p < P; p += kWarps) {
      const TreeView t = trees[p];
      const int32_t m = walk(t, s_req, n_s, g_req, len, lane, err);
      const int32_t ld = __ldg(load + p);
      if (lane == 0) out_match[b * P + p] = m;
      // Packed key: (score + 2^31) << 32 | (0xFFFF - load) << 16 | (0xFFFF - p); a larger key is a
      // better route (higher score, then lower load, then lower index).  The host guarantees
      // alpha * load <= 2^31 - 1, load <= 65535 and P <= 65536, so every field fits.
      const long long score = (long long)m - (long long)alpha * ld;
      const unsigned long long key = ((unsigned long long)(score + 2147483648LL) << 32) |
                                     ((unsigned long long)(0xFFFF - ld) << 16) | (unsigned long long)(0xFFFF - p);
      best = key > best ? key : best;
    }
    if (lane == 0) s_best[warp] = best;
    __syncthreads();
    if (threadIdx.x == 0) {
      unsigned long long k = s_best[0];
#pragma unroll
      for (int w = 1; w < kWarps; ++w) k = s_best[w] > k ? s_best[w] : k;
      out_peer[b] = 0xFFFF - (int32_t)(k & 0xFFFFull);
    }
    __syncthreads();
  }
}

}  // namespace

cudaError_t launch_route(const TreeView* d_trees, int32_t P, const int32_t* tokens, int64_t n_tokens, int64_t tok_base,
                         const int64_t* offsets, int64_t B, const int32_t* d_load, int32_t alpha, int32_t* out_match,
                         int32_t* out_peer, int32_t* d_err, int num_sms, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  const int64_t max_ctas = (int64_t)num_sms * 8;
  const int grid = (int)(B < max_ctas ? B : max_ctas);
  route_kernel<<<grid, kThreads, kSmemTokens * sizeof(int32_t), st>>>(d_trees, P, tokens, n_tokens, tok_base, offsets,
                                                                      B, d_load, alpha, out_match, out_peer, d_err);
  return cudaGetLastError();
}

}  // namespace p2p
