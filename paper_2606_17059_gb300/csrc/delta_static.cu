// delta_static.cu -- scratch for p2p_tree_apply_delta_static, the delta call that allocates nothing.
//
// Some callers cannot allocate memory when they patch their replicas: a serving loop whose device memory
// is owned by another allocator (it may not call cudaMalloc or go through a caching allocator on its hot
// path), or a process that must keep its device footprint fixed after start-up.  For them the delta call
// has a variant whose scratch -- the validation result and every op's gathered sequence -- lives in the
// one file-scope static device array below instead of router-owned buffers that grow on demand.  After the
// 256-byte header (the validation result), the array holds one done byte per op of the delta (rounded up to
// whole 4-byte words) and, only when some op's sequence is split into more than two pool runs, the gathered
// sequences: one buffer of the longest sequence per warp of the delta kernel (16 warps per tree).
//
// The array is a fixed 8 MiB + 256 B, held by every GPU that loads the library until the process exits.
// Every call shares it and it keeps the last call's contents: the header words that must start at zero
// are cleared at the start of each call.  Two calls whose device work overlaps (two routers on different
// streams, for example) race on it; callers must order such calls.
#include "internal.h"

namespace p2p {
namespace {

constexpr int64_t kHeaderInts = kStaticHeaderInts;    // 256 B: validation results
constexpr int64_t kScratchTokens = int64_t(1) << 21;  // 2,097,152 tokens = 8 MiB of gathered sequences

static __device__ __align__(256) int32_t g_delta_scratch[kHeaderInts + kScratchTokens];

}  // namespace

int64_t static_scratch_tokens() { return kScratchTokens; }

// Device address of g_delta_scratch on the current device (the caller makes the router's device current).
// In host code the array's name stands for a host-side shadow, not a device address, so the address is
// looked up on every call: the lookup allocates nothing, and a context that was torn down and created again
// (which may load the module at another address) never sees a stale pointer.  The first lookup on a device
// may load the library's module there, which is why the first call should come before any stream capture.
cudaError_t static_scratch(int device, int32_t** header, int32_t** tokens) {
  int cur = -1;
  cudaError_t e = cudaGetDevice(&cur);
  if (e != cudaSuccess) return e;
  if (cur != device) return cudaErrorInvalidDevice;
  void* p = nullptr;
  e = cudaGetSymbolAddress(&p, g_delta_scratch);
  if (e != cudaSuccess) return e;
  *header = static_cast<int32_t*>(p);
  *tokens = *header + kHeaderInts;
  return cudaSuccess;
}

}  // namespace p2p
