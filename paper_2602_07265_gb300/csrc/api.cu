// C ABI of libxshare.so (include/xshare.h): argument checks, workspace plan
// and the stream-ordered launch sequence of the MoE-layer forward.
#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>
#include <cstring>

#include "xs_internal.cuh"

namespace xs {
namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t v) { return (v + kAlign - 1) / kAlign * kAlign; }

// Per device: 0 until known, then the SM count of an sm_103 device or
// XS_ERR_DEVICE.  Filled on first use; host threads that race on it store
// the same value.
std::atomic<int> g_dev_sms[64];

// The current device's SM count, or a negative XS_ERR code.
int current_device_sms() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return XS_ERR_CUDA;
  int v = g_dev_sms[dev].load(std::memory_order_relaxed);
  if (v == 0) {
    int major = 0, minor = 0, sms = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return XS_ERR_CUDA;
    v = (major == 10 && minor == 3 && sms > 0) ? sms : XS_ERR_DEVICE;
    g_dev_sms[dev].store(v, std::memory_order_relaxed);
  }
  return v;
}

int check_route_args(int B, int N, int k, int budget, int mode, const xs_route_params *prm) {
  if (prm == nullptr) return XS_ERR_NULL;
  if (B < 1 || B > kMaxB || N < 1 || N > kMaxN || k < 1 || k > kMaxK || k > N) return XS_ERR_SHAPE;
  if (mode < XS_MODE_TOPK || mode > XS_MODE_THRESH) return XS_ERR_PARAM;
  if (mode == XS_MODE_THRESH && !(prm->tau >= 0.f && prm->tau <= 1.f)) return XS_ERR_PARAM;
  if (prm->sparse_scores != 0 && prm->sparse_scores != 1) return XS_ERR_PARAM;
  if (budget < 0 || prm->k0 < 0 || prm->k0 > kMaxK || prm->k0 > N || prm->m_r < 0 || prm->m_g < 0 ||
      prm->n_groups < 0)
    return XS_ERR_PARAM;
  if (prm->n_groups > 0 && (prm->n_groups > N || N % prm->n_groups != 0)) return XS_ERR_PARAM;
  if (mode == XS_MODE_GROUP && prm->n_groups < 1) return XS_ERR_PARAM;
  if (mode == XS_MODE_HIER &&
      (prm->tokens_per_request < 1 || prm->tokens_per_request > B || B % prm->tokens_per_request != 0))
    return XS_ERR_PARAM;
  return XS_OK;
}

int check_ffn_shape(int d, int F) {
  if (d < 128 || F < 128 || d % 128 != 0 || F % 128 != 0) return XS_ERR_SHAPE;
  if ((long long)d > (1 << 20) || (long long)F > (1 << 20)) return XS_ERR_SHAPE;
  return XS_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

template <class T>
T *at(void *ws, size_t off) {
  return reinterpret_cast<T *>(static_cast<char *>(ws) + off);
}

RouteArgs route_args(const Plan &pl, void *ws, int B, int N, int k, int budget, int mode,
                     const xs_route_params *prm) {
  RouteArgs a;
  std::memset(&a, 0, sizeof(a));
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
  a.sparse = (mode != XS_MODE_TOPK) ? prm->sparse_scores : 0;
  a.gs = at<float>(ws, pl.gs);
  a.p = at<float>(ws, pl.p);
  a.mask = at<uint8_t>(ws, pl.mask);
  a.ids = at<int32_t>(ws, pl.ids);
  a.w = at<float>(ws, pl.w);
  a.toptok = at<int32_t>(ws, pl.toptok);
  a.counts = at<int32_t>(ws, pl.counts);
  a.offsets = at<int32_t>(ws, pl.offsets);
  a.perm = at<int32_t>(ws, pl.perm);
  a.pos = at<int32_t>(ws, pl.pos);
  a.tiles = at<Tile>(ws, pl.tiles);
  a.meta = at<Meta>(ws, pl.meta);
  a.chunk_col = at<float>(ws, pl.chunk_col);
  a.chunk_marks = at<uint8_t>(ws, pl.chunk_marks);
  a.done = at<int32_t>(ws, pl.done);
  return a;
}

}  // namespace

Plan make_plan(int B, int N, int k, int d, int F, bool with_ffn, int n_sms, int n_shared) {
  Plan pl;
  std::memset(&pl, 0, sizeof(pl));
  pl.n_sms = n_sms;
  pl.max_pairs = B * k;
  pl.max_rows = B * k + n_shared * B;
  pl.max_tiles = N + (B * k) / kTileTok + 1 + n_shared * ((B + kTileTok - 1) / kTileTok);
  size_t o = 0;
  auto take = [&](size_t bytes) {
    size_t r = o;
    o = align_up(o + bytes);
    return r;
  };
  const bool split = with_ffn && B < kRouterTcMinB && d >= kRouterSplitMinD && d <= kRouterSplitMaxD;
  const int h_splits = split ? router_split_count(B, N, d, n_sms) : 1;
  pl.h = take((size_t)h_splits * B * N * 4);
  pl.p = take((size_t)B * N * 4);
  pl.mask = take((size_t)N);
  pl.ids = take((size_t)B * k * 4);
  pl.w = take((size_t)B * k * 4);
  pl.toptok = take((size_t)B * kMaxK * 4);
  pl.counts = take((size_t)N * 4);
  pl.offsets = take((size_t)(N + 1) * 4);
  pl.perm = take((size_t)B * k * 4);
  pl.pos = take((size_t)B * k * 4);
  pl.tiles = take((size_t)pl.max_tiles * sizeof(Tile));
  pl.meta = take(sizeof(Meta));
  const int chunks = (B + kChunk - 1) / kChunk;
  pl.chunk_col = take((size_t)chunks * N * 4);
  pl.chunk_marks = take((size_t)chunks * 2 * N);
  pl.done = take(4 * sizeof(int32_t));
  pl.gs = take((size_t)B * N * 4);
  if (with_ffn) {
    pl.rstat = take((size_t)(split ? router_split_ctas(B, N, d, n_sms) : router_tc_ctas(B, N, d, n_sms)) * 4);
    pl.xp = take((size_t)pl.max_rows * d * 2);
    pl.act = take((size_t)pl.max_rows * F * 2);
    pl.out = take((size_t)pl.max_rows * d * 4);
    pl.ffn_part = take(ffn_part_bytes(n_sms));
    pl.ffn_cnt = take(ffn_cnt_words(pl.max_tiles, B, d, F) * 4);
  }
  pl.total = o;
  return pl;
}

}  // namespace xs

using namespace xs;

extern "C" size_t xshare_workspace_size(int B, int N, int k, int d, int F, int mode,
                                        const xs_route_params *prm, int n_shared) {
  if (check_route_args(B, N, k, 0, mode, prm) != XS_OK) return 0;
  const bool ffn = (d != 0 || F != 0);
  if (ffn && check_ffn_shape(d, F) != XS_OK) return 0;
  if (n_shared < 0 || n_shared > kMaxShared || (!ffn && n_shared != 0)) return 0;
  const int sms = current_device_sms();
  if (sms < 0) return 0;
  return make_plan(B, N, k, d, F, ffn, sms, n_shared).total;
}

extern "C" int xshare_route(const float *scores, int B, int N, int k, int budget, int mode,
                            const xs_route_params *prm, uint8_t *sel_mask, int32_t *topk_ids,
                            float *topk_w, xs_stats *stats, int32_t *expert_counts,
                            int32_t *expert_offsets, int32_t *perm, void *workspace,
                            size_t ws_bytes, xs_stream_t stream) {
  int rc = check_route_args(B, N, k, budget, mode, prm);
  if (rc != XS_OK) return rc;
  if (!scores || !sel_mask || !topk_ids || !topk_w) return XS_ERR_NULL;
  if (!aligned16(scores)) return XS_ERR_ALIGN;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0) return XS_ERR_WORKSPACE;
  const int sms = current_device_sms();
  if (sms < 0) return sms;
  const Plan pl = make_plan(B, N, k, 0, 0, false, sms, 0);
  if (ws_bytes < pl.total) return XS_ERR_WORKSPACE;
  RouteArgs a = route_args(pl, workspace, B, N, k, budget, mode, prm);
  a.p = const_cast<float *>(scores);  // read only when logits == nullptr
  a.mask = sel_mask;
  a.ids = topk_ids;
  a.w = topk_w;
  a.stats = stats;
  a.counts_out = expert_counts;
  a.offsets_out = expert_offsets;
  a.perm_out = perm;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(a.done, 0, 3 * sizeof(int32_t), s) != cudaSuccess) return XS_ERR_CUDA;
  return launch_route(a, s) == cudaSuccess ? XS_OK : XS_ERR_CUDA;
}

namespace {

const char *const kStageNames[XS_N_STAGES] = {"router", "select", "refine", "gather", "ffn_gate_up",
                                              "ffn_down", "combine"};

}  // namespace

int xs::forward_impl(const FwdCall &c, FwdStep step) {
  const int B = c.B, d = c.d, F = c.F, N = c.N, k = c.k;
  int rc = check_route_args(B, N, k, c.budget, c.mode, c.prm);
  if (rc != XS_OK) return rc;
  rc = check_ffn_shape(d, F);
  if (rc != XS_OK) return rc;
  const bool packed = c.P_gate_up != nullptr || c.P_down != nullptr;
  const bool ep = c.ep_ranks >= 1;  // expert parallelism: this rank's FFN, no combine
  if (!c.x || !c.W_g || (!ep && !c.y)) return XS_ERR_NULL;
  if (packed ? (!c.P_gate_up || !c.P_down) : (!c.W_gate || !c.W_up || !c.W_down)) return XS_ERR_NULL;
  if (!aligned16(c.x) || !aligned16(c.W_g) || (c.y && !aligned16(c.y)) ||
      (c.scores_out && !aligned16(c.scores_out)) || (c.resid && !aligned16(c.resid)))
    return XS_ERR_ALIGN;
  if (packed ? (!aligned16(c.P_gate_up) || !aligned16(c.P_down))
             : (!aligned16(c.W_gate) || !aligned16(c.W_up) || !aligned16(c.W_down)))
    return XS_ERR_ALIGN;
  const xs_shared_experts *shared = c.shared;
  const xs_packed_experts *pshared = c.packed_shared;
  if (packed && shared && shared->n_shared != 0) return XS_ERR_PARAM;  // packed calls take packed ones
  const int n_shared = packed ? (pshared ? pshared->n : 0) : (shared ? shared->n_shared : 0);
  if (n_shared < 0 || n_shared > kMaxShared) return XS_ERR_PARAM;
  if (n_shared > 0 && !packed) {
    if (!shared->W_gate || !shared->W_up || !shared->W_down) return XS_ERR_NULL;
    if (!aligned16(shared->W_gate) || !aligned16(shared->W_up) || !aligned16(shared->W_down))
      return XS_ERR_ALIGN;
  }
  // Under expert parallelism only rank 0 computes (and reads) the shared experts.
  if (n_shared > 0 && packed && (!ep || c.ep_rank == 0)) {
    if (!pshared->gate_up || !pshared->down) return XS_ERR_NULL;
    if (!aligned16(pshared->gate_up) || !aligned16(pshared->down)) return XS_ERR_ALIGN;
  }
  void *workspace = c.workspace;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0) return XS_ERR_WORKSPACE;
  if (step == FwdStep::kCheckArgs) return XS_OK;
  const int sms = current_device_sms();
  if (sms < 0) return sms;
  const Plan pl = make_plan(B, N, k, d, F, true, sms, n_shared);
  if (c.ws_bytes < pl.total) return XS_ERR_WORKSPACE;
  if (step == FwdStep::kCheckAll) return XS_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(c.stream);
  void *const *events = c.events;

  RouteArgs a = route_args(pl, workspace, B, N, k, c.budget, c.mode, c.prm);
  float *h = at<float>(workspace, pl.h);
  a.logits = h;
  if (c.scores_out) a.p = c.scores_out;
  if (c.sel_mask) a.mask = c.sel_mask;
  if (c.topk_ids) a.ids = c.topk_ids;
  // Under expert parallelism the weights stay in the workspace for the
  // combine that follows the exchange (xshare_ep_combine); they are copied
  // out afterwards if asked for.
  if (c.topk_w && !ep) a.w = c.topk_w;
  if (ep) {
    a.ep_ranks = c.ep_ranks;
    a.ep_rank = c.ep_rank;
  }
  a.stats = c.stats;
  a.zero_words = at<int32_t>(workspace, pl.ffn_cnt);
  a.zero_count = (int)ffn_cnt_words(pl.max_tiles, B, d, F);
  a.n_shared = n_shared;

  FfnArgs f;
  std::memset(&f, 0, sizeof(f));
  f.W_gate = c.W_gate;
  f.W_up = c.W_up;
  f.W_down = c.W_down;
  f.P_gate_up = c.P_gate_up;
  f.P_down = c.P_down;
  if (n_shared > 0 && packed) {
    f.PS_gate_up = pshared->gate_up;
    f.PS_down = pshared->down;
  } else if (n_shared > 0) {
    f.S_gate = shared->W_gate;
    f.S_up = shared->W_up;
    f.S_down = shared->W_down;
  }
  f.n_shared = n_shared;
  f.xp = at<uint16_t>(workspace, pl.xp);
  f.act = at<uint16_t>(workspace, pl.act);
  f.out = at<float>(workspace, pl.out);
  f.tiles = a.tiles;
  f.meta = a.meta;
  f.stats = c.stats;
  f.part = at<void>(workspace, pl.ffn_part);
  f.cnt = at<int32_t>(workspace, pl.ffn_cnt);
  f.N = N;
  f.d = d;
  f.F = F;
  f.max_rows = pl.max_rows;
  f.max_tiles = pl.max_tiles;
  f.n_sms = sms;
  f.expert_base = ep ? c.ep_rank * (N / c.ep_ranks) : 0;

  auto mark = [&](int i) {
    return events == nullptr ||
           cudaEventRecord(reinterpret_cast<cudaEvent_t>(events[i]), s) == cudaSuccess;
  };
  if (!mark(0)) return XS_ERR_CUDA;
  cudaError_t re;
  int32_t *rstat = at<int32_t>(workspace, pl.rstat);
  a.router_status = rstat;
  if (B >= kRouterTcMinB) {
    int grid = 0;
    re = launch_router_tc(c.x, c.W_g, h, B, N, d, a.done, rstat, sms, &grid, s);
    a.router_ctas = grid;
  } else if (d < kRouterSplitMinD || d > kRouterSplitMaxD) {
    re = launch_router_logits(c.x, c.W_g, h, B, N, d, a.done, s);
    a.router_status = nullptr;
  } else {
    const int S = router_split_count(B, N, d, sms);
    re = launch_router_split(c.x, c.W_g, h, B, N, d, S, a.done, rstat, s);
    a.h_splits = S;
    a.router_ctas = router_split_ctas(B, N, d, sms);
  }
  if (re != cudaSuccess || !mark(1)) return XS_ERR_CUDA;
  a.events = events ? events + 2 : nullptr;  // between the selection and refinement kernels
  if (launch_route(a, s) != cudaSuccess || !mark(3)) return XS_ERR_CUDA;
  // The gather kernel warms L2 with the gate/up kernel's first weights once
  // the selected set is known (packed weights, without expert parallelism).
  GatherPf pf;
  std::memset(&pf, 0, sizeof(pf));
  if (packed && !ep) {
    pf.ready = a.done + 3;
    pf.mask = a.mask;
    pf.pk = static_cast<const uint8_t *>(c.P_gate_up);
    pf.N = N;
    pf.MT = F / 128;
    pf.KI = d / 64;
    pf.stage_bytes = 2 * 128 * 64 * 2;
    pf.grid = sms;
    // A refinement kernel of its own (more than kFuseChunks chunks) leaves
    // a longer window before the gate/up kernel: twice the warm-up.
    pf.pf_bytes = (B + kChunk - 1) / kChunk > kFuseChunks ? 2 * kGatherPrefetchBytes : kGatherPrefetchBytes;
  }
  if (launch_gather(c.x, a.perm, a.meta, const_cast<uint16_t *>(f.xp), ep ? f.out : nullptr,
                    pl.max_rows, B, d, k, pf, s) != cudaSuccess ||
      !mark(4))
    return XS_ERR_CUDA;
  if (launch_ffn_gate_up(f, s) != cudaSuccess || !mark(5)) return XS_ERR_CUDA;
  if (launch_ffn_down(f, s) != cudaSuccess || !mark(6)) return XS_ERR_CUDA;
  if (ep) {
    if (c.topk_w != nullptr &&
        cudaMemcpyAsync(c.topk_w, a.w, static_cast<size_t>(B) * k * sizeof(float),
                        cudaMemcpyDeviceToDevice, s) != cudaSuccess)
      return XS_ERR_CUDA;
    return XS_OK;
  }
  if (launch_combine(f.out, a.pos, a.w, a.meta, c.resid, c.y, B, d, k, n_shared, s) !=
          cudaSuccess ||
      !mark(7))
    return XS_ERR_CUDA;
  return XS_OK;
}

namespace {

FwdCall make_call(const uint16_t *x, const float *W_g, const uint16_t *W_gate,
                  const uint16_t *W_up, const uint16_t *W_down, int B, int d, int F, int N, int k,
                  int budget, int mode, const xs_route_params *prm, const xs_shared_experts *shared,
                  uint16_t *y, float *scores_out, uint8_t *sel_mask, int32_t *topk_ids,
                  float *topk_w, xs_stats *stats, void *workspace, size_t ws_bytes,
                  xs_stream_t stream, void *const *events) {
  FwdCall c;
  std::memset(&c, 0, sizeof(c));
  c.x = x;
  c.W_g = W_g;
  c.W_gate = W_gate;
  c.W_up = W_up;
  c.W_down = W_down;
  c.B = B;
  c.d = d;
  c.F = F;
  c.N = N;
  c.k = k;
  c.budget = budget;
  c.mode = mode;
  c.prm = prm;
  c.shared = shared;
  c.y = y;
  c.scores_out = scores_out;
  c.sel_mask = sel_mask;
  c.topk_ids = topk_ids;
  c.topk_w = topk_w;
  c.stats = stats;
  c.workspace = workspace;
  c.ws_bytes = ws_bytes;
  c.stream = stream;
  c.events = events;
  return c;
}

}  // namespace

extern "C" int xshare_moe_forward(const uint16_t *x, const float *W_g, const uint16_t *W_gate,
                                  const uint16_t *W_up, const uint16_t *W_down, int B, int d,
                                  int F, int N, int k, int budget, int mode,
                                  const xs_route_params *prm, const xs_shared_experts *shared,
                                  uint16_t *y, float *scores_out, uint8_t *sel_mask,
                                  int32_t *topk_ids, float *topk_w, xs_stats *stats,
                                  void *workspace, size_t ws_bytes, xs_stream_t stream) {
  return forward_impl(make_call(x, W_g, W_gate, W_up, W_down, B, d, F, N, k, budget, mode, prm,
                                shared, y, scores_out, sel_mask, topk_ids, topk_w, stats,
                                workspace, ws_bytes, stream, nullptr),
                      FwdStep::kLaunch);
}

extern "C" int xshare_moe_forward_profiled(const uint16_t *x, const float *W_g,
                                           const uint16_t *W_gate, const uint16_t *W_up,
                                           const uint16_t *W_down, int B, int d, int F, int N,
                                           int k, int budget, int mode,
                                           const xs_route_params *prm,
                                           const xs_shared_experts *shared, uint16_t *y,
                                           float *scores_out, uint8_t *sel_mask,
                                           int32_t *topk_ids, float *topk_w, xs_stats *stats,
                                           void *workspace, size_t ws_bytes, xs_stream_t stream,
                                           void *const *stage_events) {
  if (stage_events == nullptr) return XS_ERR_NULL;
  for (int i = 0; i <= XS_N_STAGES; ++i)
    if (stage_events[i] == nullptr) return XS_ERR_NULL;
  return forward_impl(make_call(x, W_g, W_gate, W_up, W_down, B, d, F, N, k, budget, mode, prm,
                                shared, y, scores_out, sel_mask, topk_ids, topk_w, stats,
                                workspace, ws_bytes, stream, stage_events),
                      FwdStep::kLaunch);
}

extern "C" int xshare_moe_forward_packed(const uint16_t *x, const float *W_g,
                                         const xs_packed_experts *experts, int B, int d, int F,
                                         int N, int k, int budget, int mode,
                                         const xs_route_params *prm,
                                         const xs_packed_experts *shared, uint16_t *y,
                                         float *scores_out, uint8_t *sel_mask, int32_t *topk_ids,
                                         float *topk_w, xs_stats *stats, void *workspace,
                                         size_t ws_bytes, xs_stream_t stream,
                                         void *const *stage_events) {
  if (experts == nullptr || experts->gate_up == nullptr || experts->down == nullptr) return XS_ERR_NULL;
  if (experts->n != N) return XS_ERR_SHAPE;
  if (stage_events != nullptr)
    for (int i = 0; i <= XS_N_STAGES; ++i)
      if (stage_events[i] == nullptr) return XS_ERR_NULL;
  FwdCall c = make_call(x, W_g, nullptr, nullptr, nullptr, B, d, F, N, k, budget, mode, prm, nullptr,
                        y, scores_out, sel_mask, topk_ids, topk_w, stats, workspace, ws_bytes, stream,
                        stage_events);
  c.P_gate_up = experts->gate_up;
  c.P_down = experts->down;
  c.packed_shared = shared;
  return forward_impl(c, FwdStep::kLaunch);
}

extern "C" int xshare_pack_experts(const uint16_t *W_gate, const uint16_t *W_up, const uint16_t *W_down,
                                   int n, int d, int F, void *gate_up, void *down, xs_stream_t stream) {
  if (n < 1 || n > kMaxN) return XS_ERR_SHAPE;
  int rc = check_ffn_shape(d, F);
  if (rc != XS_OK) return rc;
  if (!W_gate || !W_up || !W_down || !gate_up || !down) return XS_ERR_NULL;
  if (!aligned16(W_gate) || !aligned16(W_up) || !aligned16(W_down) || !aligned16(gate_up) ||
      !aligned16(down))
    return XS_ERR_ALIGN;
  const int sms = current_device_sms();
  if (sms < 0) return sms;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (launch_pack(W_gate, W_up, gate_up, n, F, d, sms, s) != cudaSuccess ||
      launch_pack(W_down, nullptr, down, n, d, F, sms, s) != cudaSuccess)
    return XS_ERR_CUDA;
  return XS_OK;
}

extern "C" int xshare_moe_forward_ep(const uint16_t *x, const float *W_g,
                                     const xs_packed_experts *local_experts, int B, int d, int F,
                                     int N, int k, int budget, int mode,
                                     const xs_route_params *prm, const xs_packed_experts *shared,
                                     int n_ranks, int rank, uint8_t *sel_mask, int32_t *topk_ids,
                                     float *topk_w, xs_stats *stats, void *workspace,
                                     size_t ws_bytes, xs_stream_t stream) {
  if (n_ranks < 1 || n_ranks > kMaxN || rank < 0 || rank >= n_ranks) return XS_ERR_PARAM;
  if (N < 1 || N % n_ranks != 0) return XS_ERR_PARAM;
  if (local_experts == nullptr || local_experts->gate_up == nullptr || local_experts->down == nullptr)
    return XS_ERR_NULL;
  if (local_experts->n != N / n_ranks) return XS_ERR_SHAPE;
  FwdCall c = make_call(x, W_g, nullptr, nullptr, nullptr, B, d, F, N, k, budget, mode, prm, nullptr,
                        nullptr, nullptr, sel_mask, topk_ids, topk_w, stats, workspace, ws_bytes,
                        stream, nullptr);
  c.P_gate_up = local_experts->gate_up;
  c.P_down = local_experts->down;
  c.packed_shared = shared;
  c.ep_ranks = n_ranks;
  c.ep_rank = rank;
  return forward_impl(c, FwdStep::kLaunch);
}

namespace {

// The plan of a forward call's workspace, after the checks xshare_ep_* share.
int ep_plan(void *workspace, int B, int N, int k, int d, int F, int mode, const xs_route_params *prm,
            int n_shared, Plan *pl) {
  int rc = check_route_args(B, N, k, 0, mode, prm);
  if (rc != XS_OK) return rc;
  rc = check_ffn_shape(d, F);
  if (rc != XS_OK) return rc;
  if (n_shared < 0 || n_shared > kMaxShared) return XS_ERR_PARAM;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) % kAlign) != 0) return XS_ERR_WORKSPACE;
  const int sms = current_device_sms();
  if (sms < 0) return sms;
  *pl = make_plan(B, N, k, d, F, true, sms, n_shared);
  return XS_OK;
}

}  // namespace

extern "C" int xshare_ep_exchange_buffer(void *workspace, int B, int N, int k, int d, int F,
                                         int mode, const xs_route_params *prm, int n_shared,
                                         float **buf, size_t *count) {
  if (buf == nullptr || count == nullptr) return XS_ERR_NULL;
  Plan pl;
  const int rc = ep_plan(workspace, B, N, k, d, F, mode, prm, n_shared, &pl);
  if (rc != XS_OK) return rc;
  *buf = at<float>(workspace, pl.out);
  *count = static_cast<size_t>(pl.max_rows) * d;
  return XS_OK;
}

extern "C" int xshare_ep_combine(void *workspace, int B, int N, int k, int d, int F, int mode,
                                 const xs_route_params *prm, int n_shared, uint16_t *y,
                                 xs_stream_t stream) {
  if (y == nullptr) return XS_ERR_NULL;
  if (!aligned16(y)) return XS_ERR_ALIGN;
  Plan pl;
  const int rc = ep_plan(workspace, B, N, k, d, F, mode, prm, n_shared, &pl);
  if (rc != XS_OK) return rc;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return launch_combine(at<float>(workspace, pl.out), at<int32_t>(workspace, pl.pos),
                        at<float>(workspace, pl.w), at<Meta>(workspace, pl.meta), nullptr, y, B, d,
                        k, n_shared, s) == cudaSuccess
             ? XS_OK
             : XS_ERR_CUDA;
}

extern "C" const char *xshare_stage_name(int i) {
  return (i >= 0 && i < XS_N_STAGES) ? kStageNames[i] : "";
}

extern "C" const char *xshare_strerror(int code) {
  switch (code) {
    case XS_OK: return "ok";
    case XS_ERR_SHAPE: return "shape out of range (B, N, k, d or F) or d/F not a multiple of 128";
    case XS_ERR_PARAM: return "invalid selection parameter (mode, budget, k0, m_r, m_g, n_groups or tokens_per_request)";
    case XS_ERR_NULL: return "a required pointer is NULL";
    case XS_ERR_WORKSPACE: return "workspace NULL, too small or not 256-byte aligned";
    case XS_ERR_ALIGN: return "a tensor pointer is not 16-byte aligned";
    case XS_ERR_CUDA: return "CUDA runtime or launch error";
    case XS_ERR_DEVICE: return "the current device is not an sm_103 (GB300) GPU";
    case XS_DEV_TIMEOUT: return "device: a bounded wait inside a kernel ran out";
    default: return "unknown xshare error code";
  }
}
