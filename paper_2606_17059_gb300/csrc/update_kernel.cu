// update_kernel.cu -- own-tree maintenance after routing: the routed batch as a device-resident INSERT delta.
//
// Algorithm 1: once request r has been sent to node k and acknowledged, the sender inserts r into its
// estimate of k's trie (UpdateTrieEstimate(r, k)); a request the node serves itself (k = its own index) goes
// into its own trie (UpdateTrie).  For a routed batch that is one INSERT per request b with peer[b] >= 0,
// into tree peer[b].  INSERTs commute (a tree is a multiset, and its canonical form depends only on the
// multiset), so the order of a tree's inserts is free: the batch is counting-sorted by tree with atomics,
// and every op is one pool run pointing at the request's tokens -- nothing is copied.  The delta kernel then
// applies it like any anti-entropy delta.
//
//   update_count_kernel    histogram of peer[] over trees (shared-memory bins when P is small), and the
//                          error bits of requests that cannot be inserted
//   update_scan_kernel     one CTA: exclusive scan of the histogram into peer_begin (int64) and the scatter
//                          cursors, total op count
//   update_scatter_kernel  op[i] = INSERT, seg_begin[i] = i, seg_off[i] / seg_len[i] = the request's tokens
#include "internal.h"

namespace p2p {
namespace {

constexpr int kUpdThreads = 256;
constexpr int kUpdSmemBins = 8192;  // trees binned in shared memory per CTA (32 KB); more go to global atomics
constexpr int kScanThreads = 1024;

// The request's token range if it can be inserted: 0 <= start <= end <= n_tokens, end - start < 2^31.
__device__ __forceinline__ bool request_range(const int64_t* offsets, int64_t b, int64_t n_tokens, int64_t& start,
                                              int64_t& len) {
  start = offsets[b];
  const int64_t end = offsets[b + 1];
  len = end - start;
  return start >= 0 && start <= end && end <= n_tokens && len <= INT32_MAX;
}

__global__ void __launch_bounds__(kUpdThreads) update_count_kernel(const int32_t* __restrict__ peer,
                                                                   const int64_t* __restrict__ offsets, int64_t B,
                                                                   int64_t n_tokens, int32_t P,
                                                                   int32_t* __restrict__ counts, int32_t* bad) {
  __shared__ int32_t s_bin[kUpdSmemBins];
  const bool smem = P <= kUpdSmemBins;
  if (smem)
    for (int32_t p = threadIdx.x; p < P; p += blockDim.x) s_bin[p] = 0;
  __syncthreads();
  int my_bad = 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < B; b += stride) {
    const int32_t k = peer[b];
    if (k < 0) continue;  // not routed: nothing to insert
    if (k >= P) {
      my_bad |= 1;
      continue;
    }
    int64_t start, len;
    if (!request_range(offsets, b, n_tokens, start, len)) {
      my_bad |= 2;
      continue;
    }
    if (smem)
      atomicAdd(&s_bin[k], 1);
    else
      atomicAdd(&counts[k], 1);
  }
  for (int o = 16; o > 0; o >>= 1) my_bad |= __shfl_xor_sync(0xffffffffu, my_bad, o);
  if ((threadIdx.x & 31) == 0 && my_bad) atomicOr(bad, my_bad);
  __syncthreads();
  if (smem)
    for (int32_t p = threadIdx.x; p < P; p += blockDim.x)
      if (s_bin[p]) atomicAdd(&counts[p], s_bin[p]);
}

// One CTA.  Thread t owns the trees [t*per, (t+1)*per): a serial sum, a block scan of the thread sums, then
// the serial scan written out.
__global__ void __launch_bounds__(kScanThreads) update_scan_kernel(const int32_t* __restrict__ counts, int32_t P,
                                                                   int64_t* __restrict__ peer_begin,
                                                                   int32_t* __restrict__ cursor,
                                                                   int64_t* __restrict__ seg_begin_end,
                                                                   int64_t* __restrict__ total) {
  __shared__ int64_t s_sum[kScanThreads];
  const int32_t per = (P + kScanThreads - 1) / kScanThreads;
  const int32_t p0 = min(P, (int32_t)threadIdx.x * per), p1 = min(P, p0 + per);
  int64_t mine = 0;
  for (int32_t p = p0; p < p1; ++p) mine += counts[p];
  s_sum[threadIdx.x] = mine;
  __syncthreads();
  for (int off = 1; off < kScanThreads; off <<= 1) {  // Hillis-Steele inclusive scan of the thread sums
    const int64_t v = threadIdx.x >= (unsigned)off ? s_sum[threadIdx.x - off] : 0;
    __syncthreads();
    s_sum[threadIdx.x] += v;
    __syncthreads();
  }
  int64_t run = s_sum[threadIdx.x] - mine;
  for (int32_t p = p0; p < p1; ++p) {
    peer_begin[p] = run;
    cursor[p] = (int32_t)run;
    run += counts[p];
  }
  if (threadIdx.x == kScanThreads - 1) {
    peer_begin[P] = s_sum[kScanThreads - 1];
    *seg_begin_end = s_sum[kScanThreads - 1];  // seg_begin[n] = n
    *total = s_sum[kScanThreads - 1];
  }
}

__global__ void __launch_bounds__(kUpdThreads) update_scatter_kernel(const int32_t* __restrict__ peer,
                                                                     const int64_t* __restrict__ offsets, int64_t B,
                                                                     int64_t n_tokens, int32_t P,
                                                                     int32_t* __restrict__ cursor,
                                                                     int32_t* __restrict__ op,
                                                                     int64_t* __restrict__ seg_begin,
                                                                     int64_t* __restrict__ seg_off,
                                                                     int32_t* __restrict__ seg_len) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < B; b += stride) {
    const int32_t k = peer[b];
    if (k < 0 || k >= P) continue;
    int64_t start, len;
    if (!request_range(offsets, b, n_tokens, start, len)) continue;
    const int32_t i = atomicAdd(&cursor[k], 1);
    op[i] = P2P_OP_INSERT;
    seg_begin[i] = i;
    seg_off[i] = start;
    seg_len[i] = (int32_t)len;
  }
}

}  // namespace

cudaError_t launch_update_count(const int32_t* peer, const int64_t* offsets, int64_t B, int64_t n_tokens, int32_t P,
                                int32_t* counts, int32_t* bad, int num_sms, cudaStream_t st) {
  const int64_t want = (B + kUpdThreads - 1) / kUpdThreads;
  const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)num_sms * 4));
  P2P_TIMED(K_UPDATE_COUNT, st,
            (update_count_kernel<<<grid, kUpdThreads, 0, st>>>(peer, offsets, B, n_tokens, P, counts, bad)));
  return cudaGetLastError();
}

cudaError_t launch_update_scan(const int32_t* counts, int32_t P, int64_t* peer_begin, int32_t* cursor,
                               int64_t* seg_begin_end, int64_t* total, cudaStream_t st) {
  P2P_TIMED(K_UPDATE_SCAN, st,
            (update_scan_kernel<<<1, kScanThreads, 0, st>>>(counts, P, peer_begin, cursor, seg_begin_end, total)));
  return cudaGetLastError();
}

cudaError_t launch_update_scatter(const int32_t* peer, const int64_t* offsets, int64_t B, int64_t n_tokens, int32_t P,
                                  int32_t* cursor, int32_t* op, int64_t* seg_begin, int64_t* seg_off, int32_t* seg_len,
                                  int num_sms, cudaStream_t st) {
  const int64_t want = (B + kUpdThreads - 1) / kUpdThreads;
  const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)num_sms * 8));
  P2P_TIMED(K_UPDATE_SCATTER, st,
            (update_scatter_kernel<<<grid, kUpdThreads, 0, st>>>(peer, offsets, B, n_tokens, P, cursor, op, seg_begin,
                                                                 seg_off, seg_len)));
  return cudaGetLastError();
}

}  // namespace p2p
