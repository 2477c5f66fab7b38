/*
 * xshare.h — C ABI of libxshare.so: one XShare MoE-layer forward on one GPU.
 *
 * XShare (arxiv 2602.07265) restricts a decode / verify batch to a set S of
 * experts chosen for the batch as a whole, by maximising the total gating
 * score of S under an expert budget (Sec. 3.2, Eq. 2), and then routes every
 * token to its top-k experts inside S (Sec. 3.4, refinement).
 *
 * Conventions for every entry point
 *   - Device pointers point to memory of the current CUDA device, row-major and
 *     contiguous, at least 16-byte aligned unless stated otherwise.  bf16
 *     tensors are passed as uint16_t (the raw bf16 bit pattern).
 *   - The caller owns every buffer.  The library does not allocate: scratch
 *     space is the caller's `workspace` of at least xshare_workspace_size()
 *     bytes, 256-byte aligned, which the calls overwrite.  Two exceptions,
 *     stated at their declarations: xshare_route_static uses a fixed array
 *     inside the library, and xshare_stack_graph_create lets CUDA allocate
 *     the graph it instantiates.
 *   - Calls are asynchronous and stream-ordered on `stream` (a cudaStream_t;
 *     NULL is the legacy default stream).  No call synchronises the stream or
 *     the device.  Two calls that share a workspace must not overlap.
 *   - Invalid arguments are detected on the host before anything is launched
 *     and returned as a negative XS_ERR_* code; nothing is written then.
 *     A failed kernel launch returns XS_ERR_CUDA.  A device-side failure (a
 *     bounded wait that ran out) is reported in xs_stats.status, which the
 *     caller reads after synchronising.
 *   - Scores must be finite (no NaN): selection compares them as fp32 values.
 *   - Host state: per-device caches of device properties (SM count, cluster
 *     occupancy) and the driver's tensor-map encoder, filled on first use and
 *     safe to fill from several host threads at once.  Calls on different
 *     workspaces and streams may run concurrently (xshare_route_static
 *     excepted, below).
 *
 * Limits: 1 <= N <= 1024 experts; 1 <= k <= min(N, 16); 0 <= k0 <= min(N, 16);
 * 1 <= B <= 8192 tokens; for the forward calls d % 128 == 0 and F % 128 == 0;
 * at most 8 shared experts.
 *
 * Entry points: xshare_route (selection and refinement on given scores) and
 * its workspace-free variant; xshare_moe_forward (the whole layer), on plain
 * or packed expert weights (xshare_pack_experts), with optional per-kernel
 * events; its expert-parallel form over several GPUs (xshare_moe_forward_ep,
 * xshare_ep_exchange_buffer, xshare_ep_combine); xshare_stack_forward and its
 * CUDA-graph form (L layers under one global budget); a bounded-wait
 * self-test; strings.
 */
#ifndef XSHARE_H
#define XSHARE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st;
/* A cudaStream_t. */
typedef struct CUstream_st *xs_stream_t;

/* Selection modes.
 *   XS_MODE_TOPK : S = E, plain top-k routing (the paper's baseline, Sec. 2.2).
 *   XS_MODE_BATCH: Algorithm 2 — warm-up S_0 = union of per-token Top k0, then
 *                  GreedySelect (Algorithm 1 with a fixed budget): the `budget`
 *                  experts of E \ S_0 with the largest column score
 *                  scores[j] = sum_i g_ij are added (Sec. 3.4).
 *   XS_MODE_GROUP: Algorithm 6 — warm-up S_0, then Algorithm 5: full rounds over
 *                  the G contiguous expert groups, each round adding every
 *                  non-exhausted group's best remaining expert, until
 *                  |S| >= m_g * G (Sec. 5, Eq. 5).
 *   XS_MODE_HIER : Algorithm 4 — per request (contiguous runs of
 *                  tokens_per_request tokens) Algorithm 3:
 *                  S_r = S0_r + Top m_r of the request's column scores; then
 *                  S = union S_r plus the `budget` best remaining experts by the
 *                  batch column score (Sec. 4, Eq. 3-4).
 *   XS_MODE_THRESH: Algorithm 2 with GreedySelect in the threshold form that
 *                  Algorithm 1 prints: warm-up S_0, then while
 *                  f(S) < tau * f(E) add the best expert of E \ S by column
 *                  score, f(S) = sum over S of the column scores (Eq. 2).
 *                  `budget` is ignored.  f(E) and f(S_0) are fp32 halving
 *                  trees over the expert index (values at their index in a
 *                  zero vector of power-of-two length, v[l] += v[l+o] for
 *                  o = len/2 .. 1); the target is the fp32 product tau * f(E);
 *                  adding e adds scores[e] to f(S) in fp32 (Proposition 1).
 * Ordering everywhere: larger score first, equal scores -> lower expert index.
 * Column scores are fp32 sums in a fixed order: rows in chunks of 32 (last one
 * zero-padded), a halving tree v[l] += v[l+o], o = 16, 8, 4, 2, 1, inside a
 * chunk, chunk sums added left to right from 0. */
enum {
  XS_MODE_TOPK = 0,
  XS_MODE_BATCH = 1,
  XS_MODE_GROUP = 2,
  XS_MODE_HIER = 3,
  XS_MODE_THRESH = 4
};

/* Selection parameters (fields a mode does not use are ignored). */
typedef struct {
  int32_t k0;                 /* warm-up: Top k0 per token (Algorithms 2, 3, 6); 0 = none */
  int32_t m_r;                /* HIER: per-request budget m_r (Algorithm 3) */
  int32_t tokens_per_request; /* HIER: 1 + L_s (Sec. 4.1); B % tokens_per_request == 0 */
  int32_t n_groups;           /* GROUP: G (Sec. 5); N % G == 0.  Also used by the
                                 max_group_load statistic in every mode; 0 = 1 */
  int32_t m_g;                /* GROUP: per-group budget m_g (Algorithm 5) */
  float tau;                  /* THRESH: covered fraction of the score mass, 0 <= tau <= 1 */
  int32_t sparse_scores;      /* 0: column scores sum the dense softmax g (default).
                                 1: they sum Sec. 2.2's top-k-masked gating values
                                 g_ij = p_ij / D_i on the token's Top k (D_i = fp32 sum
                                 of those k scores in rank order, 1/k each if D_i = 0),
                                 0 elsewhere, and an expert whose column score is 0 is
                                 never added (no gain).  Warm-up and refinement use the
                                 dense scores in both.  Ignored by TOPK. */
} xs_route_params;

/* Per-call statistics, written by the device into caller memory. */
typedef struct {
  int32_t n_selected;     /* |S| */
  int32_t n_used;         /* |U|: experts with at least one routed (token, slot) */
  int32_t union_topk;     /* |union_i Top k(G_i, E)|: experts plain top-k would activate */
  int32_t max_group_load; /* max_g |S intersect E_g| over n_groups groups (Sec. 5.1) */
  int32_t n_pairs;        /* routed (token, slot) pairs = B * min(k, |S|) */
  int32_t status;         /* 0, or an XS_DEV_* code */
  int32_t reserved[2];
} xs_stats;

/* Host-side error codes (return values). */
#define XS_OK 0
#define XS_ERR_SHAPE (-1)     /* B, N, k, d or F out of range or misaligned */
#define XS_ERR_PARAM (-2)     /* mode, budget or a field of xs_route_params invalid */
#define XS_ERR_NULL (-3)      /* a required pointer is NULL */
#define XS_ERR_WORKSPACE (-4) /* workspace NULL, too small or not 256-byte aligned */
#define XS_ERR_ALIGN (-5)     /* a tensor pointer is not 16-byte aligned */
#define XS_ERR_CUDA (-6)      /* a CUDA runtime / launch error */
#define XS_ERR_DEVICE (-7)    /* the current device is not an sm_103 (GB300) GPU */

/* Device-side status codes (xs_stats.status). */
#define XS_DEV_OK 0
#define XS_DEV_TIMEOUT 1      /* a bounded wait inside a kernel ran out */

/* Shared experts E^s_j of the layer (Sec. 2.1: y = sum_i g_i E_i(x) +
 * sum_j E^s_j(x)): every token goes through each of them with weight 1.
 * Same shapes per expert as the routed ones (d_ff = F), device pointers:
 * W_gate, W_up [n_shared, F, d] bf16; W_down [n_shared, d, F] bf16. */
typedef struct {
  const uint16_t *W_gate;
  const uint16_t *W_up;
  const uint16_t *W_down;
  int32_t n_shared;           /* 0 .. 8 */
} xs_shared_experts;

/* Expert weights packed for the FFN's weight stream (xshare_pack_experts):
 * every 128-row x 64-column tile the tensor cores consume, stored contiguously
 * in the order the kernels read it and already in the shared-memory layout
 * (128-byte swizzle), so a pipeline stage's weights arrive in one contiguous
 * bulk copy.  Same bytes as the unpacked matrices:
 *   gate_up: n * F * d * 2 bf16 (gate and up tiles interleaved),
 *   down   : n * d * F bf16.
 * Device pointers, 16-byte aligned. */
typedef struct {
  const void *gate_up;
  const void *down;
  int32_t n;                  /* experts (for shared experts: 0 .. 8) */
} xs_packed_experts;

/* Bytes of workspace the calls below need for these sizes.  For
 * xshare_route pass d = F = 0 and n_shared = 0.  Returns 0 for arguments the
 * calls would reject.  Depends on the current device's SM count. */
size_t xshare_workspace_size(int B, int N, int k, int d, int F, int mode,
                             const xs_route_params *prm, int n_shared);

/* Steps a3-a7 of the path: batch-aware selection and refinement on given scores.
 *
 *   scores   [B, N] fp32, device: gating scores g_ij (e.g. the dense softmax
 *            of the router logits, Sec. 2.2).
 *   budget   m: experts the greedy step adds beyond the warm-up set
 *            (BATCH, HIER); ignored by TOPK, GROUP and THRESH.
 *   sel_mask [N] uint8, device, out: 1 for experts in S.
 *   topk_ids [B, k] int32, device, out: per token the min(k, |S|) best experts
 *            of S, best first (Top k(G_i, S), Algorithms 2, 4, 6); unused slots -1.
 *   topk_w   [B, k] fp32, device, out: renormalised weights
 *            g_ie / D_i, D_i = fp32 sum of the routed scores in slot order
 *            (Sec. 2.2 restricted to the routed set); unused slots 0.  If
 *            D_i == 0 every routed weight is 1/min(k, |S|).
 *   stats    xs_stats, device, out, nullable.
 *   expert_counts  [N] int32, device, out, nullable: pairs routed per expert.
 *   expert_offsets [N + 1] int32, device, out, nullable: exclusive prefix sum.
 *   perm     [B * k] int32, device, out, nullable: pair ids t * k + slot grouped
 *            by expert (ascending), ascending inside an expert; the first
 *            stats.n_pairs entries are written.
 */
int xshare_route(const float *scores, int B, int N, int k, int budget, int mode,
                 const xs_route_params *prm, uint8_t *sel_mask, int32_t *topk_ids,
                 float *topk_w, xs_stats *stats, int32_t *expert_counts,
                 int32_t *expert_offsets, int32_t *perm, void *workspace,
                 size_t ws_bytes, xs_stream_t stream);

/* The whole path a1-a9: one MoE layer forward (Sec. 2.1).
 *
 *   x       [B, d] bf16, device: token hidden states.
 *   W_g     [N, d] fp32, device: router weights; h = W_g x (Sec. 2.2).
 *   W_gate  [N, F, d] bf16, device; W_up [N, F, d] bf16; W_down [N, d, F] bf16:
 *           expert e computes E_e(x) = W_down[e] (silu(W_gate[e] x) * (W_up[e] x)).
 *           Only the experts that receive a token are read.
 *   shared  nullable: shared experts, added to every token's output.
 *   y       [B, d] bf16, device, out: y_t = sum over slots of w_ts E_{ids_ts}(x_t)
 *           + sum_j E^s_j(x_t), accumulated in fp32 (routed slots in slot order,
 *           then the shared experts in order) and rounded once to bf16.
 *   scores_out [B, N] fp32, device, out, nullable: the dense softmax scores g.
 *   sel_mask, topk_ids, topk_w, stats: as in xshare_route, each nullable.
 * Other arguments as in xshare_route; the workspace size is
 * xshare_workspace_size(B, N, k, d, F, mode, prm, shared ? shared->n_shared : 0).
 */
int xshare_moe_forward(const uint16_t *x, const float *W_g, const uint16_t *W_gate,
                       const uint16_t *W_up, const uint16_t *W_down, int B, int d, int F,
                       int N, int k, int budget, int mode, const xs_route_params *prm,
                       const xs_shared_experts *shared, uint16_t *y, float *scores_out,
                       uint8_t *sel_mask, int32_t *topk_ids, float *topk_w, xs_stats *stats,
                       void *workspace, size_t ws_bytes, xs_stream_t stream);

/* xshare_route for callers that cannot allocate device memory.  The paper has
 * no counterpart: this is a deployment convenience of the library.
 *
 * Who needs it: code loaded into a host program that owns all device memory
 * through its own allocator and offers no allocation hook, and serving loops
 * that must not allocate once running (cudaMalloc can synchronise the whole
 * device).  Neither can hand xshare_route a workspace.
 *
 * Same arguments and results as xshare_route, minus the workspace.  The
 * scratch is a fixed array inside the library's device code (about 420 KB
 * on every GPU that loads the library, held until the process exits), so:
 *   - B is limited to 1024 tokens (N <= 1024 and k <= 16 as elsewhere); a
 *     larger B returns XS_ERR_SHAPE and launches nothing;
 *   - only the dense scores: prm->sparse_scores != 0 returns XS_ERR_PARAM;
 *   - the first call on a device looks up the array's device address with
 *     cudaGetSymbolAddress; make that first call before any stream capture.
 *     The address belongs to the device's current CUDA context: after a
 *     cudaDeviceReset (or any new context on the device) the next call looks
 *     it up again, so that call, too, must come before any stream capture;
 *   - every call on a device uses the same array, so calls that can overlap
 *     on the GPU (different streams, or different host threads) race and
 *     must be ordered by the caller.  Each call clears the three arrival
 *     counters it keeps in the array (a cudaMemsetAsync on `stream`); every
 *     other scratch word is written before it is read.
 * Allocates nothing (no cudaMalloc, cudaFree or allocating library call). */
int xshare_route_static(const float *scores, int B, int N, int k, int budget, int mode,
                        const xs_route_params *prm, uint8_t *sel_mask, int32_t *topk_ids,
                        float *topk_w, xs_stats *stats, int32_t *expert_counts,
                        int32_t *expert_offsets, int32_t *perm, xs_stream_t stream);

/* Kernel stages of xshare_moe_forward, in launch order: router logits,
 * selection (softmax, ranking, column scores, Algorithms 2-6), refinement
 * and permutation (inside the selection kernel for B <= 64, so its events
 * then enclose no kernel), token gather, SwiGLU gate/up, SwiGLU down,
 * weighted combine. */
#define XS_N_STAGES 7

/* xshare_moe_forward that also records CUDA events on `stream` between its
 * kernel launches, so a caller can time each stage on the launching stream:
 * stage_events[0] before the first launch and stage_events[i + 1] after
 * stage i, for i < XS_N_STAGES.  stage_events is a host array of
 * XS_N_STAGES + 1 cudaEvent_t created by the caller (not NULL).  Results are
 * identical to xshare_moe_forward. */
int xshare_moe_forward_profiled(const uint16_t *x, const float *W_g, const uint16_t *W_gate,
                                const uint16_t *W_up, const uint16_t *W_down, int B, int d,
                                int F, int N, int k, int budget, int mode,
                                const xs_route_params *prm, const xs_shared_experts *shared,
                                uint16_t *y, float *scores_out, uint8_t *sel_mask,
                                int32_t *topk_ids, float *topk_w, xs_stats *stats,
                                void *workspace, size_t ws_bytes, xs_stream_t stream,
                                void *const *stage_events);

/* Packs n experts' weights (W_gate, W_up [n, F, d], W_down [n, d, F] bf16,
 * device) into the layout of xs_packed_experts: gate_up (n F d 2 bf16) and
 * down (n d F bf16), caller-allocated device buffers that must not overlap
 * the inputs.  d, F multiples of 128.  A layout change only, done once per
 * set of weights (no counterpart in the paper).  Asynchronous on `stream`. */
int xshare_pack_experts(const uint16_t *W_gate, const uint16_t *W_up, const uint16_t *W_down, int n,
                        int d, int F, void *gate_up, void *down, xs_stream_t stream);

/* xshare_moe_forward on packed expert weights: `experts` holds the N routed
 * experts (experts->n == N), `shared` (nullable) the shared ones.  Results
 * are identical, bit for bit, to xshare_moe_forward on the unpacked weights.
 * stage_events: NULL, or XS_N_STAGES + 1 events as in
 * xshare_moe_forward_profiled. */
int xshare_moe_forward_packed(const uint16_t *x, const float *W_g, const xs_packed_experts *experts,
                              int B, int d, int F, int N, int k, int budget, int mode,
                              const xs_route_params *prm, const xs_packed_experts *shared,
                              uint16_t *y, float *scores_out, uint8_t *sel_mask, int32_t *topk_ids,
                              float *topk_w, xs_stats *stats, void *workspace, size_t ws_bytes,
                              xs_stream_t stream, void *const *stage_events);

/* Expert parallelism (Sec. 5, Eq. 5; Algorithms 5-6 choose S so that each
 * group's load is bounded): the N routed experts are split into n_ranks
 * contiguous groups E_g of N / n_ranks experts, one per GPU, and rank g holds
 * only the weights of E_g.  One layer forward over the ranks is, on every
 * rank (one process per GPU, each with its own workspace):
 *
 *   1. xshare_moe_forward_ep: router, selection, refinement and permutation
 *      over the whole batch (identical on every rank: every rank has all of x
 *      and W_g, and the kernels are deterministic), then the SwiGLU FFN of the
 *      (token, slot) pairs routed to E_g (and of the shared experts on rank
 *      0) into the rank's exchange buffer, whose other rows it sets to zero;
 *   2. the caller sums the exchange buffers of all ranks in place (an
 *      all-reduce, e.g. ncclAllReduce with ncclSum on `stream`): every row is
 *      non-zero on exactly one rank, so the sum is exact in any order;
 *   3. xshare_ep_combine: the weighted combine into y, as in
 *      xshare_moe_forward.
 *
 * xshare_moe_forward_ep
 *   local_experts  the packed weights (xshare_pack_experts) of the
 *                  local_experts->n == N / n_ranks experts of group `rank`:
 *                  experts rank * N / n_ranks ... (rank + 1) * N / n_ranks - 1.
 *   shared         nullable: the packed shared experts; the same count on every
 *                  rank, their weights read on rank 0 only (other ranks may pass
 *                  NULL pointers).
 *   n_ranks, rank  1 <= n_ranks, N % n_ranks == 0, 0 <= rank < n_ranks.
 *   sel_mask, topk_ids, topk_w, stats: as in xshare_moe_forward (nullable).
 *   Other arguments and the workspace as in xshare_moe_forward_packed.
 * xshare_ep_exchange_buffer: *buf = the exchange buffer inside `workspace`
 *   (device, fp32, *count = (B k + n_shared B) d floats: the expert output of
 *   every routed pair and shared row); the arguments are those of the forward.
 *   No GPU work.
 * xshare_ep_combine: y [B, d] bf16, device, out: the layer output from the
 *   summed exchange buffer and the routing the forward left in `workspace`;
 *   asynchronous on `stream`.
 * A rank's buffer holds its own rows as fp32 values of the rank's own FFN
 * schedule (a unit's K range may be split differently than on one GPU), so y
 * agrees with xshare_moe_forward_packed within the forward's tolerance rather
 * than bit for bit; with n_ranks == 1 it is identical. */
int xshare_moe_forward_ep(const uint16_t *x, const float *W_g, const xs_packed_experts *local_experts,
                          int B, int d, int F, int N, int k, int budget, int mode,
                          const xs_route_params *prm, const xs_packed_experts *shared, int n_ranks,
                          int rank, uint8_t *sel_mask, int32_t *topk_ids, float *topk_w,
                          xs_stats *stats, void *workspace, size_t ws_bytes, xs_stream_t stream);
int xshare_ep_exchange_buffer(void *workspace, int B, int N, int k, int d, int F, int mode,
                              const xs_route_params *prm, int n_shared, float **buf, size_t *count);
int xshare_ep_combine(void *workspace, int B, int N, int k, int d, int F, int mode,
                      const xs_route_params *prm, int n_shared, uint16_t *y, xs_stream_t stream);

/* Name of stage i of xshare_moe_forward (e.g. "router"), or "" if out of range. */
const char *xshare_stage_name(int i);

/* One MoE layer of a stack: router W_g [N, d] fp32, experts as in
 * xshare_moe_forward, optional shared experts (NULL: none), or the packed
 * forms of both.  Device pointers; several layers may point to the same
 * weights. */
typedef struct {
  const float *W_g;
  const uint16_t *W_gate;
  const uint16_t *W_up;
  const uint16_t *W_down;
  const xs_shared_experts *shared;
  const xs_packed_experts *packed;         /* nullable: packed experts, used instead of W_* */
  const xs_packed_experts *packed_shared;  /* nullable: packed shared experts (with `packed`) */
} xs_layer;

/* A stack of L MoE layers under one global expert budget (Eq. 1 at the system
 * level; the paper's practical per-layer budget m_l = K / L, Sec. 3.2):
 *
 *   x_{l+1} = x_l + MoE_l(x_l),   l = 0 .. L-1,   x_0 = x,
 *
 * where MoE_l is xshare_moe_forward with layer l's weights and selection
 * budget m_l = floor(K_total / L) + (l < K_total mod L ? 1 : 0), so that the
 * budgets sum to K_total (used by BATCH and HIER; the other modes take no
 * budget).  The sum x_l + MoE_l(x_l) is accumulated in fp32 (x_l first) and
 * rounded once to bf16.
 *
 *   x      [B, d] bf16, device: the input of layer 0.
 *   layers host array of L xs_layer (1 <= L <= 4096).
 *   h_out  [L, B, d] bf16, device, out: h_out[l] = x_{l+1}; must not overlap x.
 *   stats  [L] xs_stats, device, out, nullable: layer l's statistics.
 *   workspace: xshare_workspace_size(B, N, k, d, F, mode, prm, n) bytes with n
 *          the largest shared-expert count of the layers; the layers run one
 *          after another on `stream` and reuse it.
 * Every layer's arguments are checked before the first launch.  The call
 * launches 6 or 7 kernels per layer and may be captured into a CUDA graph by
 * the caller; xshare_stack_graph_create does that itself. */
int xshare_stack_forward(const uint16_t *x, const xs_layer *layers, int L, int B, int d, int F,
                         int N, int k, int K_total, int mode, const xs_route_params *prm,
                         uint16_t *h_out, xs_stats *stats, void *workspace, size_t ws_bytes,
                         xs_stream_t stream);

/* A CUDA graph of one xshare_stack_forward call (opaque). */
typedef struct xs_graph xs_graph;

/* Captures xshare_stack_forward with these arguments into a CUDA graph on a
 * private stream and instantiates it; *out receives the handle (NULL on
 * error).  Nothing runs on the GPU.  The graph keeps every device pointer and
 * the host values of `layers`, `prm` and the shared-expert descriptors as
 * they are now: replays read and write the same buffers, which must stay
 * allocated until xshare_stack_graph_destroy.  CUDA allocates host and device
 * resources for the graph itself. */
int xshare_stack_graph_create(const uint16_t *x, const xs_layer *layers, int L, int B, int d,
                              int F, int N, int k, int K_total, int mode,
                              const xs_route_params *prm, uint16_t *h_out, xs_stats *stats,
                              void *workspace, size_t ws_bytes, xs_graph **out);

/* Replays the graph on `stream` (asynchronous).  Replays that share a
 * workspace or outputs must not overlap. */
int xshare_stack_graph_launch(xs_graph *g, xs_stream_t stream);

/* Releases the graph (NULL is ignored).  No replay may be pending. */
void xshare_stack_graph_destroy(xs_graph *g);

/* Self-test of the library's failure reporting (no counterpart in the paper).
 * Launches one kernel that waits, through the same bounded wait every
 * pipeline wait of the library uses, on a barrier that nothing arrives at.
 * After `budget_ns` nanoseconds (1 .. 2e9) the wait gives up; the kernel
 * writes XS_DEV_TIMEOUT to stats->status, the milliseconds it waited to
 * stats->reserved[0], and returns, leaving the CUDA context usable.
 * stats: device pointer (not NULL).  Asynchronous on `stream`. */
int xshare_selftest_wait_timeout(xs_stats *stats, uint64_t budget_ns, xs_stream_t stream);

/* A static string describing an XS_ERR_* or XS_DEV_* code (never NULL). */
const char *xshare_strerror(int code);

#ifdef __cplusplus
}
#endif

#endif /* XSHARE_H */
