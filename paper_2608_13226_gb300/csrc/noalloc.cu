// coverprune_knn_noalloc: the neighbour entry point for callers that cannot
// allocate device memory.
//
// Some callers hold no device allocator at all: a host runtime that hands
// the library only its own input and output buffers (for instance an
// inference server whose memory pool is fixed and sealed at start-up, or a
// plugin loaded into a process whose allocations are owned by someone
// else).  coverprune_knn needs a caller-provided workspace for its per-scene
// scratch; this variant keeps that scratch in a fixed array compiled into
// the library instead, so the caller passes only inputs and outputs.
//
// The scratch is one status block (256 bytes) plus one 64-byte per-scene
// record for at most kNoAllocMaxScenes scenes: 65,792 bytes, held by every
// GPU that loads the library until the process exits.  Every call shares
// it; the per-scene records are fully rewritten by each call before they are
// read, so nothing from an earlier call leaks into a later one, but two
// calls whose work overlaps on the GPU (different streams, or different host
// threads on one device) race on it.
#include <mutex>

#include "internal.h"

namespace cp {
namespace {

constexpr int64_t kNoAllocMaxScenes = 1024;
constexpr size_t kNoAllocStatusBytes = 256;
constexpr size_t kNoAllocBytes = kNoAllocStatusBytes + sizeof(SceneStats) * kNoAllocMaxScenes;

// Device address of the scratch array, found once per device.
std::mutex g_noalloc_mu;
void* g_noalloc_addr[64];

}  // namespace

static __device__ __align__(256) unsigned char g_knn_scratch[kNoAllocBytes];

// The name g_knn_scratch is only a host-side stand-in for the array: a
// kernel must be given the device address, which cudaGetSymbolAddress
// returns for the current device.  The first call on each device does this
// look-up (a runtime query, no allocation) and caches the result.
static int noalloc_scratch(void** out) {
  int dev = 0;
  CP_TRY_STATUS(cuda_status(cudaGetDevice(&dev), "coverprune_knn_noalloc: current device"));
  if (dev < 0 || dev >= 64) return CP_EUNSUPPORTED;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (g_noalloc_addr[dev] == nullptr) {
    void* p = nullptr;
    CP_TRY_STATUS(cuda_status(cudaGetSymbolAddress(&p, g_knn_scratch),
                              "coverprune_knn_noalloc: scratch address"));
    g_noalloc_addr[dev] = p;
  }
  *out = g_noalloc_addr[dev];
  return CP_OK;
}

}  // namespace cp

using namespace cp;

extern "C" int coverprune_knn_noalloc(const float* pos, int64_t B, int64_t N, int64_t k,
                                      int32_t* nbr, float* diameter, cp_stream_t stream) {
  if (B < 0 || N < 0 || B > 65535 || k < 0 || (N > 0 && k > N - 1)) return CP_EINVAL;
  if (B == 0 || N == 0) return CP_OK;
  if (B > kNoAllocMaxScenes) {
    note_message("coverprune_knn_noalloc: more scenes than the fixed scratch holds (1024)");
    return CP_EUNSUPPORTED;
  }
  if (N > kMaxKnnN) return CP_EUNSUPPORTED;
  if (!pos || ((uintptr_t)pos % 4) != 0 || (k > 0 && (!nbr || ((uintptr_t)nbr % 4) != 0)) ||
      (diameter && ((uintptr_t)diameter % 4) != 0))
    return CP_EINVAL;
  int64_t L = 2;
  while (L < k) L <<= 1;
  if (8 * L + 4 * N > 200 * 1024) return CP_EUNSUPPORTED;
  void* scratch = nullptr;
  CP_TRY_STATUS(noalloc_scratch(&scratch));
  cudaStream_t s = (cudaStream_t)stream;
  unsigned char* base = static_cast<unsigned char*>(scratch);
  SceneStats* stats = reinterpret_cast<SceneStats*>(base + kNoAllocStatusBytes);
  // the status word must start at zero; the per-scene records are rewritten
  // by the first kernel below
  CP_TRY_STATUS(cuda_status(cudaMemsetAsync(base, 0, sizeof(int), s),
                            "coverprune_knn_noalloc: status"));
  CP_TRY_STATUS(launch_scene_stats(pos, nullptr, B, N, stats, s));
  CP_TRY_STATUS(launch_knn(pos, nullptr, B, N, (int)k, k > 0 ? nbr : nullptr, stats, s));
  if (diameter) CP_TRY_STATUS(launch_diameter(stats, B, diameter, s));
  return CP_OK;
}
