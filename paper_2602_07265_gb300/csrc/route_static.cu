// xshare_route_static: the selection / refinement / permutation of
// xshare_route for callers that cannot allocate device memory.
//
// Some hosts own every byte of device memory through their own allocator and
// give the code they load no way to allocate more; some serving loops must
// not allocate after start-up because cudaMalloc can synchronise the device.
// Such callers cannot supply xshare_route's workspace.  This entry point
// keeps its scratch in a fixed array that the library module itself defines
// in device memory, sized for at most kStaticMaxB tokens, so the caller passes
// only its inputs and outputs.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <cstring>
#include <mutex>

#include "xs_internal.cuh"

namespace xs {
namespace {

constexpr int kStaticMaxB = 1024;
constexpr size_t kStaticAlign = 256;

constexpr size_t up256(size_t v) { return (v + kStaticAlign - 1) / kStaticAlign * kStaticAlign; }

constexpr int kStaticMaxPairs = kStaticMaxB * kMaxK;
constexpr int kStaticMaxTiles = kMaxN + kStaticMaxPairs / kTileTok + 1;

// Scratch layout (byte offsets), sized for B <= kStaticMaxB, N <= kMaxN, k <= kMaxK.
constexpr size_t kOffTopTok = 0;
constexpr size_t kOffCounts = kOffTopTok + up256(sizeof(int32_t) * kStaticMaxB * kMaxK);
constexpr size_t kOffOffsets = kOffCounts + up256(sizeof(int32_t) * kMaxN);
constexpr size_t kOffPerm = kOffOffsets + up256(sizeof(int32_t) * (kMaxN + 1));
constexpr size_t kOffPos = kOffPerm + up256(sizeof(int32_t) * kStaticMaxPairs);
constexpr size_t kOffTiles = kOffPos + up256(sizeof(int32_t) * kStaticMaxPairs);
constexpr size_t kOffMeta = kOffTiles + up256(sizeof(Tile) * kStaticMaxTiles);
constexpr int kStaticChunks = (kStaticMaxB + kChunk - 1) / kChunk;
constexpr size_t kOffChunkCol = kOffMeta + up256(sizeof(Meta));
constexpr size_t kOffChunkMarks = kOffChunkCol + up256(sizeof(float) * kStaticChunks * kMaxN);
constexpr size_t kOffDone = kOffChunkMarks + up256(static_cast<size_t>(kStaticChunks) * 2 * kMaxN);
constexpr size_t kStaticBytes = kOffDone + up256(4 * sizeof(int32_t));

// The scratch itself: one copy per device that loads the library, kept until
// the process exits.  From host code this name is only a handle for
// cudaGetSymbolAddress, never a device address.
static __device__ __align__(256) unsigned char g_route_scratch[kStaticBytes];

constexpr int kMaxDevices = 64;

// Where g_route_scratch lives on a device, valid for one CUDA context of that
// device: a cudaDeviceReset destroys the primary context and with it the
// module's copy of the array, and the next context loads a new copy at
// another address.  The address is therefore kept with the unique id of the
// context it was looked up in and looked up again when the current context
// has another id.  The mutex makes the set-up safe when host threads race
// on it.
struct ScratchAddr {
  std::mutex mu;
  unsigned long long ctx_id = 0;
  bool valid = false;
  void *addr = nullptr;
};
ScratchAddr g_scratch[kMaxDevices];

// The driver's cuCtxGetCurrent and cuCtxGetId, through the runtime's entry
// point query (the library does not link libcuda).  Function-local statics
// are initialised once even when threads race on the first call.
template <class Fn>
Fn driver_fn(const char *name, int version) {
  void *ptr = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &ptr, version, cudaEnableDefault, &q) == cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    return reinterpret_cast<Fn>(ptr);
  return nullptr;
}

// Id of the context current on this thread; false if there is none.
bool current_context_id(unsigned long long *id) {
  static const PFN_cuCtxGetCurrent_v4000 get_current =
      driver_fn<PFN_cuCtxGetCurrent_v4000>("cuCtxGetCurrent", 4000);
  static const PFN_cuCtxGetId_v12000 get_id = driver_fn<PFN_cuCtxGetId_v12000>("cuCtxGetId", 12000);
  if (get_current == nullptr || get_id == nullptr) return false;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return false;
  return get_id(ctx, id) == CUDA_SUCCESS;
}

// Device address of g_route_scratch in the current context of device `dev`
// (the current device), or nullptr on a CUDA error.  The look-up runs on the
// first call in each context of the device; later calls reuse it.
void *scratch_address(int dev) {
  ScratchAddr &slot = g_scratch[dev];
  std::lock_guard<std::mutex> lock(slot.mu);
  unsigned long long id = 0;
  if (slot.valid && current_context_id(&id) && id == slot.ctx_id) return slot.addr;
  // Set-up: cudaGetSymbolAddress also makes the device's primary context
  // current if no context was yet.
  void *addr = nullptr;
  if (cudaGetSymbolAddress(&addr, g_route_scratch) != cudaSuccess || addr == nullptr) return nullptr;
  if (!current_context_id(&id)) return nullptr;
  slot.addr = addr;
  slot.ctx_id = id;
  slot.valid = true;
  return addr;
}

}  // namespace
}  // namespace xs

using namespace xs;

extern "C" int xshare_route_static(const float *scores, int B, int N, int k, int budget, int mode,
                                   const xs_route_params *prm, uint8_t *sel_mask,
                                   int32_t *topk_ids, float *topk_w, xs_stats *stats,
                                   int32_t *expert_counts, int32_t *expert_offsets,
                                   int32_t *perm, xs_stream_t stream) {
  if (prm == nullptr) return XS_ERR_NULL;
  if (B < 1 || B > kStaticMaxB || N < 1 || N > kMaxN || k < 1 || k > kMaxK || k > N)
    return XS_ERR_SHAPE;
  if (mode < XS_MODE_TOPK || mode > XS_MODE_THRESH) return XS_ERR_PARAM;
  if (mode == XS_MODE_THRESH && !(prm->tau >= 0.f && prm->tau <= 1.f)) return XS_ERR_PARAM;
  if (prm->sparse_scores != 0) return XS_ERR_PARAM;  // the dense reading only
  if (budget < 0 || prm->k0 < 0 || prm->k0 > kMaxK || prm->k0 > N || prm->m_r < 0 ||
      prm->m_g < 0 || prm->n_groups < 0)
    return XS_ERR_PARAM;
  if (prm->n_groups > 0 && (prm->n_groups > N || N % prm->n_groups != 0)) return XS_ERR_PARAM;
  if (mode == XS_MODE_GROUP && prm->n_groups < 1) return XS_ERR_PARAM;
  if (mode == XS_MODE_HIER &&
      (prm->tokens_per_request < 1 || prm->tokens_per_request > B || B % prm->tokens_per_request != 0))
    return XS_ERR_PARAM;
  if (!scores || !sel_mask || !topk_ids || !topk_w) return XS_ERR_NULL;
  if ((reinterpret_cast<uintptr_t>(scores) & 15u) != 0) return XS_ERR_ALIGN;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return XS_ERR_CUDA;
  int major = 0, minor = 0;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
    return XS_ERR_CUDA;
  if (major != 10 || minor != 3) return XS_ERR_DEVICE;
  char *base = static_cast<char *>(scratch_address(dev));
  if (base == nullptr) return XS_ERR_CUDA;

  RouteArgs a;
  std::memset(&a, 0, sizeof(a));
  a.p = const_cast<float *>(scores);  // read only: no logits are given
  a.B = B;
  a.N = N;
  a.k = k;
  a.budget = budget;
  a.mode = mode;
  a.k0 = (mode == XS_MODE_TOPK) ? 0 : prm->k0;
  a.m_r = prm->m_r;
  a.T = prm->tokens_per_request < 1 ? 1 : prm->tokens_per_request;
  a.G = prm->n_groups < 1 ? 1 : prm->n_groups;
  a.m_g = prm->m_g > N ? N : prm->m_g;
  a.tau = prm->tau;
  a.mask = sel_mask;
  a.ids = topk_ids;
  a.w = topk_w;
  a.toptok = reinterpret_cast<int32_t *>(base + kOffTopTok);
  a.counts = reinterpret_cast<int32_t *>(base + kOffCounts);
  a.offsets = reinterpret_cast<int32_t *>(base + kOffOffsets);
  a.perm = reinterpret_cast<int32_t *>(base + kOffPerm);
  a.pos = reinterpret_cast<int32_t *>(base + kOffPos);
  a.tiles = reinterpret_cast<Tile *>(base + kOffTiles);
  a.meta = reinterpret_cast<Meta *>(base + kOffMeta);
  a.stats = stats;
  a.counts_out = expert_counts;
  a.offsets_out = expert_offsets;
  a.perm_out = perm;
  a.chunk_col = reinterpret_cast<float *>(base + kOffChunkCol);
  a.chunk_marks = reinterpret_cast<uint8_t *>(base + kOffChunkMarks);
  a.done = reinterpret_cast<int32_t *>(base + kOffDone);
  a.zero_words = nullptr;
  a.zero_count = 0;
  // The three arrival counters must start at zero; every other scratch word is
  // written before it is read.
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(a.done, 0, 3 * sizeof(int32_t), s) != cudaSuccess) return XS_ERR_CUDA;
  return launch_route(a, s) == cudaSuccess ? XS_OK : XS_ERR_CUDA;
}
