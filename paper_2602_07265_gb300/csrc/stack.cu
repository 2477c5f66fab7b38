// A stack of L residual MoE layers under one global expert budget (Eq. 1 at
// the system level), launched stream-ordered or replayed from a CUDA graph.
//
// Layer l computes x_{l+1} = x_l + MoE_l(x_l) with the single-layer path
// (router, selection, refinement, permutation, expert FFN, combine); the
// residual add happens in the combine kernel, before the one rounding to
// bf16.  The selection budget of layer l is the uniform split of K
// (Sec. 3.2: m_l = K / L), as integers that sum to K.  Layers run one after
// the other on the caller's stream and share one workspace.
#include <cuda_runtime.h>

#include <cstdint>
#include <cstring>
#include <new>

#include "xs_internal.cuh"

struct xs_graph {
  cudaGraph_t graph;
  cudaGraphExec_t exec;
};

namespace xs {
namespace {

constexpr int kMaxLayers = 4096;

int layer_budget(int K, int L, int l) { return K / L + (l < K % L ? 1 : 0); }

// The call of layer l.
FwdCall layer_call(const uint16_t *x, const xs_layer *layers, int L, int l, int B, int d, int F,
                   int N, int k, int K_total, int mode, const xs_route_params *prm,
                   uint16_t *h_out, xs_stats *stats, void *workspace, size_t ws_bytes,
                   xs_stream_t stream) {
  FwdCall c;
  std::memset(&c, 0, sizeof(c));
  const size_t act = static_cast<size_t>(B) * d;
  c.x = l == 0 ? x : h_out + (l - 1) * act;
  c.resid = c.x;
  c.y = h_out + l * act;
  c.W_g = layers[l].W_g;
  c.W_gate = layers[l].W_gate;
  c.W_up = layers[l].W_up;
  c.W_down = layers[l].W_down;
  c.shared = layers[l].shared;
  if (layers[l].packed != nullptr) {
    c.W_gate = c.W_up = c.W_down = nullptr;
    c.P_gate_up = layers[l].packed->gate_up;
    c.P_down = layers[l].packed->down;
    c.packed_shared = layers[l].packed_shared;
    c.shared = nullptr;
  }
  c.B = B;
  c.d = d;
  c.F = F;
  c.N = N;
  c.k = k;
  c.budget = layer_budget(K_total, L, l);
  c.mode = mode;
  c.prm = prm;
  c.stats = stats ? stats + l : nullptr;
  c.workspace = workspace;
  c.ws_bytes = ws_bytes;
  c.stream = stream;
  return c;
}

bool overlaps(const void *a, size_t na, const void *b, size_t nb) {
  const uintptr_t pa = reinterpret_cast<uintptr_t>(a), pb = reinterpret_cast<uintptr_t>(b);
  return pa < pb + nb && pb < pa + na;
}

// Checks every layer (its arguments, then the device and the workspace) and,
// with `launch`, runs them; a rejected call launches nothing.
int stack_run(const uint16_t *x, const xs_layer *layers, int L, int B, int d, int F, int N, int k,
              int K_total, int mode, const xs_route_params *prm, uint16_t *h_out,
              xs_stats *stats, void *workspace, size_t ws_bytes, xs_stream_t stream, bool launch) {
  if (L < 1 || L > kMaxLayers) return XS_ERR_SHAPE;
  if (K_total < 0) return XS_ERR_PARAM;
  if (!layers || !x || !h_out) return XS_ERR_NULL;
  if (B >= 1 && d >= 1) {
    const size_t act = static_cast<size_t>(B) * d * 2;
    if (overlaps(x, act, h_out, act * L)) return XS_ERR_PARAM;
  }
  for (int l = 0; l < L; ++l)
    if (layers[l].packed != nullptr && layers[l].packed->n != N) return XS_ERR_SHAPE;
  for (FwdStep step : {FwdStep::kCheckArgs, FwdStep::kCheckAll, FwdStep::kLaunch}) {
    if (step == FwdStep::kLaunch && !launch) break;
    for (int l = 0; l < L; ++l) {
      const int rc = forward_impl(layer_call(x, layers, L, l, B, d, F, N, k, K_total, mode, prm,
                                             h_out, stats, workspace, ws_bytes, stream),
                                  step);
      if (rc != XS_OK) return rc;
    }
  }
  return XS_OK;
}

}  // namespace
}  // namespace xs

using namespace xs;

extern "C" int xshare_stack_forward(const uint16_t *x, const xs_layer *layers, int L, int B,
                                    int d, int F, int N, int k, int K_total, int mode,
                                    const xs_route_params *prm, uint16_t *h_out, xs_stats *stats,
                                    void *workspace, size_t ws_bytes, xs_stream_t stream) {
  return stack_run(x, layers, L, B, d, F, N, k, K_total, mode, prm, h_out, stats, workspace,
                   ws_bytes, stream, true);
}

extern "C" int xshare_stack_graph_create(const uint16_t *x, const xs_layer *layers, int L, int B,
                                         int d, int F, int N, int k, int K_total, int mode,
                                         const xs_route_params *prm, uint16_t *h_out,
                                         xs_stats *stats, void *workspace, size_t ws_bytes,
                                         xs_graph **out) {
  if (out == nullptr) return XS_ERR_NULL;
  *out = nullptr;
  int rc = stack_run(x, layers, L, B, d, F, N, k, K_total, mode, prm, h_out, stats, workspace,
                     ws_bytes, nullptr, false);
  if (rc != XS_OK) return rc;
  cudaStream_t s = nullptr;
  if (cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking) != cudaSuccess) return XS_ERR_CUDA;
  cudaGraph_t graph = nullptr;
  if (cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
    rc = XS_ERR_CUDA;
  } else {
    rc = stack_run(x, layers, L, B, d, F, N, k, K_total, mode, prm, h_out, stats, workspace,
                   ws_bytes, reinterpret_cast<xs_stream_t>(s), true);
    const cudaError_t e = cudaStreamEndCapture(s, &graph);
    if (rc == XS_OK && e != cudaSuccess) rc = XS_ERR_CUDA;
  }
  cudaGraphExec_t exec = nullptr;
  if (rc == XS_OK && cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess) rc = XS_ERR_CUDA;
  cudaStreamDestroy(s);
  xs_graph *g = nullptr;
  if (rc == XS_OK) {
    g = new (std::nothrow) xs_graph;
    if (g == nullptr) rc = XS_ERR_CUDA;
  }
  if (rc != XS_OK) {
    if (exec) cudaGraphExecDestroy(exec);
    if (graph) cudaGraphDestroy(graph);
    return rc;
  }
  g->graph = graph;
  g->exec = exec;
  *out = g;
  return XS_OK;
}

extern "C" int xshare_stack_graph_launch(xs_graph *g, xs_stream_t stream) {
  if (g == nullptr) return XS_ERR_NULL;
  return cudaGraphLaunch(g->exec, reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? XS_OK
             : XS_ERR_CUDA;
}

extern "C" void xshare_stack_graph_destroy(xs_graph *g) {
  if (g == nullptr) return;
  cudaGraphExecDestroy(g->exec);
  cudaGraphDestroy(g->graph);
  delete g;
}
