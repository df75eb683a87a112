// delta_static.cu -- scratch for p2p_tree_apply_delta_static, the delta call that allocates nothing.
//
// Some callers cannot allocate memory when they patch their replicas: a serving loop whose device memory
// is owned by another allocator (it may not call cudaMalloc or go through a caching allocator on its hot
// path), or a process that must keep its device footprint fixed after start-up.  For them the delta call
// has a variant whose scratch -- the validation result and every op's gathered sequence -- lives in the
// one file-scope static device array below instead of router-owned buffers that grow on demand.
//
// The array is a fixed 8 MiB + 256 B, held by every GPU that loads the library until the process exits.
// Every call shares it and it keeps the last call's contents: the header words that must start at zero
// are cleared at the start of each call.  Two calls whose device work overlaps (two routers on different
// streams, for example) race on it; callers must order such calls.
#include <mutex>

#include "internal.h"

namespace p2p {
namespace {

constexpr int64_t kHeaderInts = 64;                   // 256 B: validation results
constexpr int64_t kScratchTokens = int64_t(1) << 21;  // 2,097,152 tokens = 8 MiB of gathered sequences

static __device__ __align__(256) int32_t g_delta_scratch[kHeaderInts + kScratchTokens];

// Header (int32 words): [0..1] longest sequence (u64), [2] error bits (StaticCheck).

__global__ void validate_kernel(const int32_t* __restrict__ op, const int64_t* __restrict__ seg_begin,
                                const int64_t* __restrict__ seg_off, const int32_t* __restrict__ seg_len, int64_t n,
                                int64_t n_segs, int64_t n_pool, const int64_t* __restrict__ peer_begin, int32_t P) {
  unsigned long long* max_len = reinterpret_cast<unsigned long long*>(g_delta_scratch);
  int32_t* err = g_delta_scratch + 2;
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
      atomicMax(max_len, (unsigned long long)len);
    }
    if (bits) atomicOr(err, bits);
  }
  if (peer_begin && blockIdx.x == 0) {
    for (int32_t p = threadIdx.x; p <= P; p += blockDim.x) {
      const int64_t v = peer_begin[p];
      if ((p == 0 && v != 0) || (p == P && v != n) || (p > 0 && v < peer_begin[p - 1]))
        atomicOr(err, STATIC_BAD_PEER_BEGIN);
    }
  }
}

// Sets each tree's op range for this call on the device (peer_begin stays in device memory).
__global__ void init_ranges_kernel(TreeState* states, int32_t nt, const int64_t* __restrict__ peer_begin, int64_t n) {
  const int32_t i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= nt) return;
  states[i].op_next = peer_begin ? peer_begin[i] : 0;
  states[i].op_end = peer_begin ? peer_begin[i + 1] : n;
  states[i].status = DELTA_OK;
  states[i].n_absent = 0;
}

std::mutex g_addr_mutex;
void* g_addr[256] = {};

}  // namespace

int64_t static_scratch_tokens() { return kScratchTokens; }

// Device address of g_delta_scratch.  Looked up once per device, by the first call that runs with that
// device current (the caller makes the router's device current); the result is cached per device.
cudaError_t static_scratch(int device, int32_t** header, int32_t** tokens) {
  if (device < 0 || device >= 256) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_addr_mutex);
  if (!g_addr[device]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_delta_scratch);
    if (e != cudaSuccess) return e;
    g_addr[device] = p;
  }
  *header = static_cast<int32_t*>(g_addr[device]);
  *tokens = *header + kHeaderInts;
  return cudaSuccess;
}

// Clears the header, then validates the (device-resident) delta into it.
cudaError_t launch_validate_static(int32_t* header, const p2p_delta* d, int32_t peer, int32_t P, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(header, 0, kHeaderInts * sizeof(int32_t), st);
  if (e != cudaSuccess) return e;
  const p2p_seqs& S = d->seqs;
  const int64_t blocks = std::min<int64_t>((S.n + 255) / 256, 4096);
  validate_kernel<<<(int)std::max<int64_t>(blocks, 1), 256, 0, st>>>(d->op, S.seg_begin, S.seg_off, S.seg_len, S.n,
                                                                    S.n_segs, S.n_pool,
                                                                    peer == -1 ? d->peer_begin : nullptr, P);
  return cudaGetLastError();
}

cudaError_t launch_init_ranges(TreeState* d_states, int32_t nt, const int64_t* peer_begin, int64_t n, cudaStream_t st) {
  init_ranges_kernel<<<(nt + 127) / 128, 128, 0, st>>>(d_states, nt, peer_begin, n);
  return cudaGetLastError();
}

}  // namespace p2p
