// Internal declarations shared by the translation units of libxshare.so.
#pragma once

#include <cuda_runtime.h>
#include <cstddef>
#include <cstdint>
#include <utility>

#include "xshare.h"

namespace xs {

// Programmatic dependent launch.  Every kernel of the library is launched
// with programmatic stream serialization and calls pdl_wait(), which returns
// once all work before it in the stream has completed and is visible, and
// only after that pdl_trigger(), so that the next kernel's CTAs may be
// scheduled while this one runs (they block in their own pdl_wait()).  Every
// CTA waits before it exits.  Hence when a CTA of kernel n starts, kernel
// n - 2 and everything before it have completed: the FFN kernels read the
// routing results (written two or more launches earlier) and start their
// weight loads before pdl_wait(), and the combine kernel reads its rows,
// weights and x_t then; every other access to global memory, in every
// kernel, comes after it.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launches `kernel` on `s` with programmatic stream serialization allowed.
template <class... Params, class... Args>
cudaError_t launch_pdl(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

constexpr int kMaxN = 1024;     // experts
constexpr int kMaxK = 16;       // top-k and warm-up k0
constexpr int kMaxB = 8192;     // tokens
constexpr int kTileTok = 128;   // tokens of one expert handled by one FFN tile
constexpr int kRouteThreads = 1024;
constexpr int kChunk = 32;                   // tokens per selection CTA (= the column-sum chunk)
constexpr int kScatterMaxN = 256;            // parallel stable scatter up to this many experts
constexpr int kFuseChunks = 2;               // up to this many chunks the selection CTA also refines
constexpr int kMaxShared = 8;                // shared experts
constexpr int kGatherPrefetchBytes = 256 * 1024;  // L2 warm-up per gate/up CTA (packed weights)
constexpr int kGatherWarmBlocks = 32;              // gather blocks that issue the warm-up

// CTAs an FFN kernel splits its U units (a token tile x 128 weight rows, KI
// K steps each) over, at most `grid`.  Stream-K gives CTA c the steps
// [I c / G, I (c + 1) / G) of I = U KI, at least kFfnMinSteps each; a unit
// cut between CTAs is finished from partial sums.  When q = ceil(U / grid)
// is 1 or 2, divides U, and G = U / q CTAs still cover 80 % of the SMs, G is
// that: every range then ends on a unit boundary and no unit is cut (no
// partial sums, no reductions), which measured OLMoE B = 8 at 58.7 -> 52.5 us
// on GB300.  With more units per CTA or more idle SMs the cuts cost less
// than the longer per-CTA stream (DeepSeek-R1 B = 8 on 81 % of the SMs, five
// units each: 398 -> 409 us).  The gather kernel's L2 warm-up predicts the
// gate/up split with the same function.
constexpr int kFfnMinSteps = 8;
__host__ __device__ inline int ffn_ctas(long long U, int KI, int grid) {
  const long long I = U * KI, want = (I + kFfnMinSteps - 1) / kFfnMinSteps;
  const long long q = (U + grid - 1) / grid;
  if (U > 0 && q <= 2 && U % q == 0 && (U / q) * 5 >= static_cast<long long>(grid) * 4)
    return static_cast<int>(U / q);
  return static_cast<int>(want < grid ? want : grid);
}

// One FFN work tile: up to kTileTok consecutive rows of the permuted pair
// list, all routed to `expert`.  Experts N .. N + n_shared - 1 are the shared
// experts; their rows follow the routed pairs: row n_pairs + j * B + t is
// token t's pass through shared expert j.
struct Tile {
  int32_t expert;
  int32_t row0;
  int32_t ntok;
  int32_t pad;
};

// Device-side facts of one call, written by the routing kernel and read by
// the kernels after it (so that no host synchronisation is needed).
struct Meta {
  int32_t n_pairs;      // B * k'
  int32_t n_tiles;      // FFN tiles
  int32_t kprime;       // k' = min(k, |S|)
  int32_t n_selected;
  int32_t n_used;
  int32_t union_topk;
  int32_t max_group_load;
  int32_t status;       // XS_DEV_*
  int32_t n_rows;       // FFN rows: n_pairs + n_shared * B
  // The FFN work of this call: routed tiles [ffn_t0, ffn_t1) and shared-expert
  // tiles [ffn_s0, ffn_s1), in that order; the rows they write: routed rows
  // [row0, row1) and, if srows, the shared rows.  Without expert parallelism
  // that is every tile and row; with it, those of the rank's expert group.
  int32_t ffn_t0, ffn_t1, ffn_s0, ffn_s1;
  int32_t row0, row1, srows;
};

// Byte offsets of every workspace region (256-byte aligned).
struct Plan {
  size_t h, p, mask, ids, w, toptok, counts, offsets, perm, pos, tiles, meta;
  size_t chunk_col, chunk_marks, done, gs, rstat;
  size_t xp, act, out, ffn_part, ffn_cnt;
  size_t total;
  int max_pairs;   // routed pairs B * k
  int max_rows;    // FFN rows: routed pairs plus n_shared * B
  int max_tiles, n_sms;
};

Plan make_plan(int B, int N, int k, int d, int F, bool with_ffn, int n_sms, int n_shared);

struct RouteArgs {
  const float *logits;   // nullable: if set, p = softmax(logits) is computed first
  int h_splits;          // logits as h_splits slices [h_splits][B][N], added in slice order
  float *p;              // [B, N] scores (input if logits == nullptr, else output)
  int B, N, k, budget, mode, k0, m_r, T, G, m_g;
  float tau;             // THRESH: covered fraction of the score mass
  int sparse;            // column scores from the top-k-masked gating values
  float *gs;             // [B, N] those values, written when HIER needs them from global
  uint8_t *mask;         // [N]
  int32_t *ids;          // [B, k]
  float *w;              // [B, k]
  int32_t *toptok;       // [B, 16] per-token ranked top over E
  int32_t *counts;       // [N]
  int32_t *offsets;      // [N + 1]
  int32_t *perm;         // [B * k]
  int32_t *pos;          // [B * k] inverse of perm (row of pair t*k+s), -1 if unrouted
  Tile *tiles;           // [max_tiles]
  Meta *meta;
  xs_stats *stats;       // nullable
  int32_t *counts_out;   // nullable caller copies
  int32_t *offsets_out;
  int32_t *perm_out;
  float *chunk_col;      // [C][N] column-sum tree of each 32-token chunk
  uint8_t *chunk_marks;  // [C][2][N] each chunk's warm-up / base marks and union marks
  int32_t *done;         // [4] arrival counters (selection, refinement, union), zero at
                         // entry, and the selected-set flag (done[3])
  int32_t *zero_words;   // nullable: region cleared for the FFN kernels
  int zero_count;
  void *const *events;   // nullable: events[0] is recorded between the two kernels
  int fuse_refine;       // set by launch_route: refinement runs in the selection kernel
  int n_shared;          // shared-expert tiles appended after the routed ones
  const int32_t *router_status;  // nullable: per-CTA status of the tensor-core router
  int router_ctas;
  int ep_ranks, ep_rank;  // expert parallelism: the FFN work of group ep_rank of ep_ranks (0: all)
};

cudaError_t launch_route(const RouteArgs &a, cudaStream_t s);
// Router logits for B < kRouterTcMinB.  d outside [kRouterSplitMinD,
// kRouterSplitMaxD]: whole-d blocks of 8 tokens x 4 experts (route.cu),
// h[t][e].  d inside: d-sliced blocks (router_split.cu), h[s][t][e] for s <
// router_split_count(), one slice of d each, which the selection kernel
// adds in order; status: [router_split_ctas()] words, one per CTA.
constexpr int kRouterSplitMinD = 4096;
constexpr int kRouterSplitMaxD = 16384;
cudaError_t launch_router_logits(const uint16_t *x, const float *Wg, float *h, int B, int N,
                                 int d, int32_t *done, cudaStream_t s);
int router_split_count(int B, int N, int d, int n_sms);
int router_split_ctas(int B, int N, int d, int n_sms);
cudaError_t launch_router_split(const uint16_t *x, const float *Wg, float *h, int B, int N, int d,
                                int S, int32_t *done, int32_t *status, cudaStream_t s);
// The router on the tensor cores (router_tc.cu).  status: [router_tc_ctas()]
// words, an upper bound on its grid; each launched CTA writes its word.
constexpr int kRouterTcMinB = 64;   // batches from this size use it
int router_tc_ctas(int B, int N, int d, int n_sms);
cudaError_t launch_router_tc(const uint16_t *x, const float *Wg, float *h, int B, int N, int d,
                             int32_t *done, int32_t *status, int n_sms, int *grid_out,
                             cudaStream_t s);
cudaError_t launch_combine(const float *out, const int32_t *pos, const float *w,
                           const Meta *meta, const uint16_t *resid, uint16_t *y, int B, int d,
                           int k, int n_shared, cudaStream_t s);
// Gathers the token rows of this call's FFN rows into xp; with expert
// parallelism (zero_out != nullptr) it zeroes the rows of zero_out that
// another rank computes.
// What the gather kernel needs to warm L2 with the gate/up kernel's first
// weights (packed weights only; pk == nullptr: no warm-up).
struct GatherPf {
  const int32_t *ready;   // done[3]: set by the selection kernel once the mask is written
  const uint8_t *mask;    // [N] selected set
  const uint8_t *pk;      // packed gate/up weights
  int N, MT, KI;          // experts; the gate/up kernel's row blocks and K steps per unit
  int stage_bytes;        // packed bytes per step (gate and up tiles)
  int grid;               // the gate/up kernel's grid
  int pf_bytes;           // bytes per gate/up CTA to prefetch
};
cudaError_t launch_gather(const uint16_t *x, const int32_t *perm, const Meta *meta,
                          uint16_t *xp, float *zero_out, int max_rows, int B, int d, int k,
                          const GatherPf &pf, cudaStream_t s);

struct FfnArgs {
  const uint16_t *W_gate, *W_up, *W_down;
  const uint16_t *S_gate, *S_up, *S_down;   // shared experts, used when n_shared > 0
  // Packed weights (pack.cu), nullable; when set they replace the matrices above.
  const void *P_gate_up, *P_down, *PS_gate_up, *PS_down;
  int n_shared;
  const uint16_t *xp;    // [max_rows, d] permuted token rows
  uint16_t *act;         // [max_rows, F] silu(g) * u, bf16
  float *out;            // [max_rows, d] expert outputs, fp32
  const Tile *tiles;
  Meta *meta;
  xs_stats *stats;       // nullable
  void *part;            // partial-sum scratch
  int32_t *cnt;          // arrival counters (cleared by the routing kernel)
  int N, d, F, max_rows, max_tiles, n_sms;
  int expert_base;       // routed expert e uses weights e - expert_base (expert parallelism)
};

cudaError_t launch_ffn_gate_up(const FfnArgs &a, cudaStream_t s);
cudaError_t launch_ffn_down(const FfnArgs &a, cudaStream_t s);
size_t ffn_part_bytes(int n_sms);
// Packs W0 (and W1) [n][M][K] bf16 into 128 x 64 swizzled tiles (pack.cu).
cudaError_t launch_pack(const uint16_t *W0, const uint16_t *W1, void *P, int n, int M, int K,
                        int n_sms, cudaStream_t s);
size_t ffn_cnt_words(int max_tiles, int B, int d, int F);

// One MoE-layer forward as the C entry points describe it, plus `resid`
// (nullable): x_t added to y_t before rounding.
struct FwdCall {
  const uint16_t *x;
  const float *W_g;
  const uint16_t *W_gate, *W_up, *W_down;
  int B, d, F, N, k, budget, mode;
  const xs_route_params *prm;
  const xs_shared_experts *shared;
  const uint16_t *resid;
  const void *P_gate_up, *P_down;          // nullable: packed weights instead of W_gate/W_up/W_down
  const xs_packed_experts *packed_shared;  // nullable: packed shared experts
  uint16_t *y;
  float *scores_out;
  uint8_t *sel_mask;
  int32_t *topk_ids;
  float *topk_w;
  xs_stats *stats;
  void *workspace;
  size_t ws_bytes;
  xs_stream_t stream;
  void *const *events;
  int ep_ranks, ep_rank;  // > 1: expert parallelism; the call ends after the FFN (no combine)
};

enum class FwdStep {
  kCheckArgs,   // host-side argument checks only (no CUDA call)
  kCheckAll,    // also the device and the workspace size
  kLaunch,      // check everything, then launch
};
int forward_impl(const FwdCall &c, FwdStep step);

}  // namespace xs
