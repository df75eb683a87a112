// delta_static.cu -- scratch for p2p_tree_apply_delta_static, the delta call that allocates nothing.
//
// Some callers cannot allocate memory when they patch their replicas: a serving loop whose device memory
// is owned by another allocator (it may not call cudaMalloc or go through a caching allocator on its hot
// path), or a process that must keep its device footprint fixed after start-up.  For them the delta call
// has a variant whose scratch -- the validation result and every op's gathered sequence -- lives in the
// one file-scope static device array below instead of router-owned buffers that grow on demand.  After the
// header, the array holds one cursor per (tree, bucket) of the delta kernel and, only for ops whose
// sequence is split into more than two pool runs, the gathered sequences.
//
// The array is a fixed 8 MiB + 256 B, held by every GPU that loads the library until the process exits.
// Every call shares it and it keeps the last call's contents: the header words that must start at zero
// are cleared at the start of each call.  Two calls whose device work overlaps (two routers on different
// streams, for example) race on it; callers must order such calls.
#include <mutex>

#include "internal.h"

namespace p2p {
namespace {

constexpr int64_t kHeaderInts = kStaticHeaderInts;    // 256 B: validation results
constexpr int64_t kScratchTokens = int64_t(1) << 21;  // 2,097,152 tokens = 8 MiB of gathered sequences

static __device__ __align__(256) int32_t g_delta_scratch[kHeaderInts + kScratchTokens];

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

}  // namespace p2p
