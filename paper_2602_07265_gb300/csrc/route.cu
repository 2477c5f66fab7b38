// Router, batch-aware expert selection, refinement, permutation, gather and
// combine kernels (steps a1-a7 and a9 of the MoE-layer forward).
//
// Selection follows XShare (arxiv 2602.07265): Algorithm 2 (BATCH),
// Algorithms 3-4 (HIER), Algorithms 5-6 (GROUP) and plain top-k (TOPK), on
// fp32 gating scores, with the refinement "route x_i to Top k(G_i, S)" and
// the renormalised weights of Sec. 2.2.
#include <cuda_bf16.h>

#include <climits>
#include <cmath>

#include "xs_internal.cuh"

namespace xs {
namespace {

constexpr unsigned kFull = 0xffffffffu;

// Order-preserving 32-bit key of an fp32 score (larger score -> larger key;
// -0 is read as +0 so that equal scores get equal keys).  Key 0 marks "no
// candidate": no finite score maps to it.
__device__ __forceinline__ uint32_t score_key(float v) {
  if (v == 0.f) v = 0.f;
  const uint32_t u = __float_as_uint(v);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float key_score(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// Canonical fp32 sum of p[r, col] over rows r in [r0, r1): chunks of 32 rows
// (zero padded), halving tree inside a chunk, chunk sums added left to right
// from 0 (Algorithm 1 / Eq. 2 with a fixed summation order).
__device__ __forceinline__ float canonical_sum(const float *__restrict__ p, int N, int col,
                                               int r0, int r1) {
  float acc = 0.f;
  for (int c0 = r0; c0 < r1; c0 += 32) {
    float v[32];
#pragma unroll
    for (int l = 0; l < 32; ++l) v[l] = (c0 + l < r1) ? p[(size_t)(c0 + l) * N + col] : 0.f;
#pragma unroll
    for (int o = 16; o; o >>= 1) {
#pragma unroll
      for (int l = 0; l < o; ++l) v[l] = __fadd_rn(v[l], v[l + o]);
    }
    acc = __fadd_rn(acc, v[0]);
  }
  return acc;
}

// ---------------------------------------------------------------------------
// Warp-wide ranking.  A warp ranks up to 32 Q candidates: lane l holds the
// candidates l + 32 q (q < Q) as (key, index) pairs, sorted best first in
// registers by a bitonic network; each round then takes the best head of all
// lanes with two warp reductions (largest key, then smallest index among the
// lanes holding it) and the winning lane pops its head.
template <int Q>
struct LaneList {
  uint32_t key[Q];
  int idx[Q];
};

// Total order of every top-k and argmax: larger score first, equal scores ->
// lower expert index.
__device__ __forceinline__ bool before(uint32_t ka, int ia, uint32_t kb, int ib) {
  return ka > kb || (ka == kb && ia < ib);
}

template <int Q>
__device__ __forceinline__ void lane_sort(LaneList<Q> &L) {
#pragma unroll
  for (int k = 2; k <= Q; k <<= 1) {
#pragma unroll
    for (int j = k >> 1; j > 0; j >>= 1) {
#pragma unroll
      for (int i = 0; i < Q; ++i) {
        const int l = i ^ j;
        if (l > i) {
          const bool first_best = (i & k) == 0;
          const bool sw = first_best ? before(L.key[l], L.idx[l], L.key[i], L.idx[i])
                                     : before(L.key[i], L.idx[i], L.key[l], L.idx[l]);
          if (sw) {
            const uint32_t tk = L.key[i];
            L.key[i] = L.key[l];
            L.key[l] = tk;
            const int ti = L.idx[i];
            L.idx[i] = L.idx[l];
            L.idx[l] = ti;
          }
        }
      }
    }
  }
}

// Takes up to `count` candidates best first, calling emit(r, index, score)
// on every lane; returns how many were taken.
template <int Q, class Emit>
__device__ __forceinline__ int lane_take(LaneList<Q> &L, int count, Emit emit) {
  int r = 0;
  for (; r < count; ++r) {
    const uint32_t mx = __reduce_max_sync(kFull, L.key[0]);
    if (mx == 0u) break;
    const uint32_t cand = (L.key[0] == mx) ? static_cast<uint32_t>(L.idx[0]) : 0xffffffffu;
    const int win = static_cast<int>(__reduce_min_sync(kFull, cand));
    emit(r, win, key_score(mx));
    if (L.key[0] == mx && L.idx[0] == win) {
#pragma unroll
      for (int q = 0; q + 1 < Q; ++q) {
        L.key[q] = L.key[q + 1];
        L.idx[q] = L.idx[q + 1];
      }
      L.key[Q - 1] = 0u;
    }
  }
  return r;
}

// Loads candidates j = j0 + lane + 32 q in [j0, j0 + n) with keys from
// `val(q, j)` where `live(q, j)` holds.
template <int Q, class Val, class Live>
__device__ __forceinline__ void lane_load(LaneList<Q> &L, int j0, int n, int lane, Val val,
                                          Live live) {
#pragma unroll
  for (int q = 0; q < Q; ++q) {
    const int j = j0 + lane + 32 * q;
    L.idx[q] = j;
    L.key[q] = (lane + 32 * q < n && live(q, j)) ? score_key(val(q, j)) : 0u;
  }
}

// Exclusive block-wide scan of three ints per thread; returns the totals.
__device__ __forceinline__ void block_scan3(int (&v)[3], int (&tot)[3], int *s_tmp /*[32][3]*/) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int inc[3] = {v[0], v[1], v[2]};
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
#pragma unroll
    for (int c = 0; c < 3; ++c) {
      const int t = __shfl_up_sync(kFull, inc[c], o);
      if (lane >= o) inc[c] += t;
    }
  }
  if (lane == 31)
#pragma unroll
    for (int c = 0; c < 3; ++c) s_tmp[warp * 3 + c] = inc[c];
  __syncthreads();
  if (warp == 0) {
#pragma unroll
    for (int c = 0; c < 3; ++c) {
      const int x = lane < nw ? s_tmp[lane * 3 + c] : 0;
      int y = x;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(kFull, y, o);
        if (lane >= o) y += t;
      }
      s_tmp[96 + lane * 3 + c] = y - x;  // exclusive prefix of warp totals
      if (lane == 31) s_tmp[192 + c] = y;
    }
  }
  __syncthreads();
#pragma unroll
  for (int c = 0; c < 3; ++c) {
    v[c] = inc[c] - v[c] + s_tmp[96 + warp * 3 + c];
    tot[c] = s_tmp[192 + c];
  }
  __syncthreads();
}

// The whole selection in one CTA (steps a2-a7):
//   1. per token (one warp each): dense softmax of the logits (or the given
//      scores), then its ranked top-max(k, k0) over E, which marks the plain
//      top-k union and the warm-up set S_0;
//   2. canonical column sums (one thread per expert) and, for HIER, the
//      per-request selections of Algorithm 3 (one warp per request);
//   3. the budgeted selection: BATCH and the batch step of HIER rank the
//      column scores outside the base set in one warp; GROUP ranks each
//      group's scores in its own warp (Algorithm 5's rounds in closed form);
//   4. per token the top-k' inside S with renormalised weights, counting the
//      pairs per expert on the way;
//   5. prefix sums, FFN tiles, and the stable scatter of the pairs.
// The score matrix and the ids are staged in shared memory when they fit.
template <int kQ>
__global__ void __launch_bounds__(kRouteThreads, 1) route_kernel(RouteArgs a) {
  extern __shared__ float dsm[];
  __shared__ uint8_t s_mask[kMaxN];   // S
  __shared__ uint8_t s_base[kMaxN];   // S_0 (or the union of the S_r for HIER)
  __shared__ uint8_t s_union[kMaxN];  // union of plain top-k
  __shared__ float s_col[kMaxN];      // batch column scores
  __shared__ int32_t s_counts[kMaxN];
  __shared__ int32_t s_cursor[kMaxN];
  __shared__ int32_t s_avail[kMaxN];
  __shared__ int32_t s_tmp[200];
  __shared__ int32_t s_scal[8];       // 0:R* 1:max group load 2:|U| 3:tiles 4:pairs

  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = blockDim.x >> 5;
  const int B = a.B, N = a.N, k = a.k;
  const int kk = max(k, a.k0);  // ranked list length per token
  const bool hier = a.mode == XS_MODE_HIER;
  float *ps = a.p_smem ? dsm : nullptr;
  int32_t *ids_s = a.ids_smem ? reinterpret_cast<int32_t *>(dsm + (a.p_smem ? B * N : 0)) : nullptr;
  // Per-warp expert counts of the parallel scatter: [32][N] after p and ids.
  int32_t *s_wcnt = reinterpret_cast<int32_t *>(dsm) + (a.p_smem ? B * N : 0) + (a.ids_smem ? B * k : 0);
  const float *P = ps ? ps : a.p;

  for (int j = tid; j < N; j += blockDim.x) {
    s_mask[j] = 0;
    s_base[j] = 0;
    s_union[j] = 0;
    s_counts[j] = 0;
  }
  if (a.zero_words != nullptr)
    for (int i = tid; i < a.zero_count; i += blockDim.x) a.zero_words[i] = 0;
  __syncthreads();

  // ---- 1. scores (a2) and per-token ranking over E (a3) ----
  for (int t = warp; t < B; t += nwarps) {
    float vals[kQ];
    if (a.logits != nullptr) {
      const float *hrow = a.logits + (size_t)t * N;
      float mx = -INFINITY;
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        const int j = lane + 32 * q;
        vals[q] = (j < N) ? hrow[j] : -INFINITY;
        mx = fmaxf(mx, vals[q]);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, o));
      float sum = 0.f;
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        vals[q] = (lane + 32 * q < N) ? expf(vals[q] - mx) : 0.f;
        sum = __fadd_rn(sum, vals[q]);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) sum = __fadd_rn(sum, __shfl_xor_sync(kFull, sum, o));
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        const int j = lane + 32 * q;
        if (j < N) {
          vals[q] = __fdiv_rn(vals[q], sum);
          a.p[(size_t)t * N + j] = vals[q];
          if (ps) ps[t * N + j] = vals[q];
        }
      }
    } else {
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        const int j = lane + 32 * q;
        vals[q] = (j < N) ? a.p[(size_t)t * N + j] : 0.f;
        if (ps && j < N) ps[t * N + j] = vals[q];
      }
    }
    LaneList<kQ> L;
    lane_load<kQ>(L, 0, N, lane, [&](int q, int) { return vals[q]; },
                  [](int, int) { return true; });
    lane_sort<kQ>(L);
    int32_t *top = a.toptok + (size_t)t * kMaxK;
    lane_take<kQ>(L, kk, [&](int r, int id, float) {
      if (lane == 0) {
        if (r < k) s_union[id] = 1;
        if (r < a.k0) {
          if (hier)
            top[r] = id;
          else
            s_base[id] = 1;
        }
      }
    });
  }
  __syncthreads();

  // ---- 2. batch column scores (a4) ----
  for (int j = tid; j < N; j += blockDim.x) s_col[j] = canonical_sum(P, N, j, 0, B);

  // ---- 2'. HIER: per-request selection (Algorithm 3), one warp per request ----
  if (hier) {
    const int T = a.T, R = B / T;
    for (int r = warp; r < R; r += nwarps) {
      const int r0 = r * T, r1 = r0 + T;
      float sc[kQ];
      uint32_t excl = 0;
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        const int j = lane + 32 * q;
        sc[q] = (j < N) ? canonical_sum(P, N, j, r0, r1) : 0.f;
      }
      // S0_r: union of Top k0 over the request's tokens.
      for (int x = r0; x < r1; ++x)
        for (int i = 0; i < a.k0; ++i) {
          const int e = a.toptok[(size_t)x * kMaxK + i];
          if ((unsigned)e < (unsigned)N && (e & 31) == lane) {
            excl |= 1u << (e >> 5);
            s_base[e] = 1;
          }
        }
      // S_r = S0_r + Top m_r(scores_r, E \ S0_r).
      LaneList<kQ> L;
      lane_load<kQ>(L, 0, N, lane, [&](int q, int) { return sc[q]; },
                    [&](int q, int) { return ((excl >> q) & 1u) == 0; });
      lane_sort<kQ>(L);
      lane_take<kQ>(L, a.m_r, [&](int, int id, float) {
        if (lane == 0) s_base[id] = 1;
      });
    }
  }
  __syncthreads();

  // ---- 3. budgeted selection (a5) ----
  for (int j = tid; j < N; j += blockDim.x) s_mask[j] = s_base[j];
  __syncthreads();
  if (a.mode == XS_MODE_TOPK) {
    for (int j = tid; j < N; j += blockDim.x) s_mask[j] = 1;
  } else if (a.mode == XS_MODE_GROUP) {
    // Algorithm 5 runs whole rounds; after R rounds group g has added
    // min(R, avail_g) of its best remaining experts.  R* is the first round
    // count reaching m_g * G, or the one that exhausts every group.
    const int G = a.G, size = N / G;
    const int n_base = __syncthreads_count(tid < N && s_base[tid]);
    for (int g = warp; g < G; g += nwarps) {
      int c = 0;
      for (int j = g * size + lane; j < (g + 1) * size; j += 32) c += s_base[j] ? 0 : 1;
      c = __reduce_add_sync(kFull, c);
      if (lane == 0) s_avail[g] = c;
    }
    __syncthreads();
    if (tid == 0) {
      int maxav = 0;
      for (int g = 0; g < G; ++g) maxav = max(maxav, s_avail[g]);
      const long long target = (long long)a.m_g * G;
      int R = 0;
      for (;;) {
        long long tot = n_base;
        for (int g = 0; g < G; ++g) tot += min(R, s_avail[g]);
        if (tot >= target || R >= maxav) break;
        ++R;
      }
      s_scal[0] = R;
    }
    __syncthreads();
    const int R = s_scal[0];
    if (R > 0)
      for (int g = warp; g < G; g += nwarps) {
        LaneList<kQ> L;
        lane_load<kQ>(L, g * size, size, lane, [&](int, int j) { return s_col[j]; },
                      [&](int, int j) { return s_base[j] == 0; });
        lane_sort<kQ>(L);
        lane_take<kQ>(L, R, [&](int, int id, float) {
          if (lane == 0) s_mask[id] = 1;
        });
      }
  } else if (warp == 0) {
    // BATCH (Algorithm 2) and the batch step of HIER (Algorithm 4): add the
    // `budget` best experts outside the base set by the batch column score.
    LaneList<kQ> L;
    lane_load<kQ>(L, 0, N, lane, [&](int, int j) { return s_col[j]; },
                  [&](int, int j) { return s_base[j] == 0; });
    lane_sort<kQ>(L);
    __syncwarp();
    lane_take<kQ>(L, a.budget, [&](int, int id, float) {
      if (lane == 0) s_mask[id] = 1;
    });
  }
  __syncthreads();

  // ---- statistics ----
  const int nsel = __syncthreads_count(tid < N && s_mask[tid]);
  const int n_union = __syncthreads_count(tid < N && s_union[tid]);
  if (warp == 0) {
    const int G = a.G >= 1 ? a.G : 1;
    const int size = N / G;
    int best = 0;
    for (int g = lane; g < G; g += 32) {
      int c = 0;
      for (int j = g * size; j < (g + 1) * size; ++j) c += s_mask[j];
      best = max(best, c);
    }
    best = __reduce_max_sync(kFull, best);
    if (lane == 0) s_scal[1] = best;
  }
  for (int j = tid; j < N; j += blockDim.x) a.mask[j] = s_mask[j];
  const int kp = min(k, nsel);

  // ---- 4. refinement (a6): Top k'(G_i, S), renormalised weights, pair counts ----
  for (int t = warp; t < B; t += nwarps) {
    LaneList<kQ> L;
    const float *prow = P + (size_t)t * N;
    lane_load<kQ>(L, 0, N, lane, [&](int, int j) { return prow[j]; },
                  [&](int, int j) { return s_mask[j] != 0; });
    lane_sort<kQ>(L);
    int my_id = -1;  // lane s keeps slot s
    float my_v = 0.f;
    float D = 0.f;
    const int got = lane_take<kQ>(L, kp, [&](int r, int id, float v) {
      if (lane == r) {
        my_id = id;
        my_v = v;
      }
      D = __fadd_rn(D, v);  // slot order, identical on every lane
    });
    if (lane < k) {
      float wv = 0.f;
      if (lane < got) wv = (D > 0.f) ? __fdiv_rn(my_v, D) : __fdiv_rn(1.f, (float)got);
      const int id = (lane < got) ? my_id : -1;
      a.ids[(size_t)t * k + lane] = id;
      a.w[(size_t)t * k + lane] = wv;
      if (ids_s) ids_s[t * k + lane] = id;
      if (id >= 0) atomicAdd(&s_counts[id], 1);
    }
  }
  __syncthreads();

  // ---- 5. permutation (a7): counting sort by expert, stable in (token, slot) ----
  {
    const int c = tid < N ? s_counts[tid] : 0;
    int v[3] = {c, (c + kTileTok - 1) / kTileTok, c > 0 ? 1 : 0}, tot[3];
    block_scan3(v, tot, s_tmp);
    if (tid < N) {
      s_cursor[tid] = v[0];
      a.counts[tid] = c;
      a.offsets[tid] = v[0];
      if (a.counts_out) a.counts_out[tid] = c;
      if (a.offsets_out) a.offsets_out[tid] = v[0];
      for (int tt = 0; tt * kTileTok < c; ++tt) {
        Tile tl;
        tl.expert = tid;
        tl.row0 = v[0] + tt * kTileTok;
        tl.ntok = min(kTileTok, c - tt * kTileTok);
        tl.pad = 0;
        a.tiles[v[1] + tt] = tl;
      }
    }
    if (tid == 0) {
      a.offsets[N] = tot[0];
      if (a.offsets_out) a.offsets_out[N] = tot[0];
      s_scal[2] = tot[2];
      s_scal[3] = tot[1];
      s_scal[4] = tot[0];
    }
  }
  __syncthreads();
  const int P2 = B * k;
  const int32_t *ids = ids_s ? ids_s : a.ids;
  if (N <= kScatterMaxN) {
    // Chunks of blockDim pairs: rank inside a warp by match_any, then an
    // exclusive prefix over the warps of the chunk for every expert.
    const unsigned lt = (1u << lane) - 1u;
    for (int base = 0; base < P2; base += blockDim.x) {
      for (int i = tid; i < 32 * N; i += blockDim.x) s_wcnt[i] = 0;
      const int q = base + tid;
      int e = (q < P2) ? ids[q] : -1;
      if ((unsigned)e >= (unsigned)N) e = -1;
      const unsigned peers = __match_any_sync(kFull, e);
      const int rank = __popc(peers & lt);
      __syncthreads();
      if (e >= 0 && rank == 0) s_wcnt[warp * N + e] = __popc(peers);
      __syncthreads();
      if (tid < N) {
        int run = 0;
        for (int w = 0; w < nwarps; ++w) {
          const int x = s_wcnt[w * N + tid];
          s_wcnt[w * N + tid] = run;
          run += x;
        }
        s_avail[tid] = run;
      }
      __syncthreads();
      if (e >= 0) {
        const int r = s_cursor[e] + s_wcnt[warp * N + e] + rank;
        a.perm[r] = q;
        a.pos[q] = r;
        if (a.perm_out) a.perm_out[r] = q;
      } else if (q < P2) {
        a.pos[q] = -1;
      }
      __syncthreads();
      if (tid < N) s_cursor[tid] += s_avail[tid];
      __syncthreads();
    }
  } else if (warp == 0) {
    const unsigned lt = (1u << lane) - 1u;
    for (int base = 0; base < P2; base += 32) {
      const int q = base + lane;
      int e = (q < P2) ? ids[q] : -1;
      if ((unsigned)e >= (unsigned)N) e = -1;
      const unsigned peers = __match_any_sync(kFull, e);
      const int rank = __popc(peers & lt);
      const int old = (e >= 0) ? s_cursor[e] : 0;
      __syncwarp();
      if (e >= 0) {
        const int r = old + rank;
        a.perm[r] = q;
        a.pos[q] = r;
        if (a.perm_out) a.perm_out[r] = q;
        if (rank == 0) s_cursor[e] = old + __popc(peers);
      } else if (q < P2) {
        a.pos[q] = -1;
      }
      __syncwarp();
    }
  }
  if (tid == 0) {
    Meta m;
    m.n_pairs = s_scal[4];  // == B * kp unless scores were non-finite
    m.n_tiles = s_scal[3];
    m.kprime = kp;
    m.n_selected = nsel;
    m.n_used = s_scal[2];
    m.union_topk = n_union;
    m.max_group_load = s_scal[1];
    m.status = 0;
    for (int i = 0; i < 8; ++i) m.pad[i] = 0;
    *a.meta = m;
    if (a.stats) {
      xs_stats st;
      st.n_selected = nsel;
      st.n_used = s_scal[2];
      st.union_topk = n_union;
      st.max_group_load = s_scal[1];
      st.n_pairs = s_scal[4];
      st.status = 0;
      st.reserved[0] = st.reserved[1] = 0;
      *a.stats = st;
    }
  }
}

// ---- a1: router logits h = W_g x, fp32.
// A block owns 8 tokens x 4 experts; its 8 warps split the d dimension into
// 8 contiguous slices.  A lane walks its slice in float4 steps, keeping the
// 8 x 4 outer-product sums in registers, with the next step's x and W_g
// values loaded before the current step's FMAs.  A butterfly reduce-scatter
// over the 32 lanes leaves each lane one finished sum, and the 8 warp
// partials are added in warp order through shared memory: a fixed order, so
// h is reproducible bit for bit.
constexpr int kRtTok = 8;
constexpr int kRtExp = 4;
constexpr int kRtWarps = 8;
constexpr int kRtOut = kRtTok * kRtExp;   // 32 sums per lane before the reduction

__device__ __forceinline__ void rt_load(const uint2 *__restrict__ xbase,
                                        const float4 *__restrict__ wbase, int t0, int e0, int B,
                                        int N, int d4, int c4, uint2 (&xv)[kRtTok],
                                        float4 (&wv)[kRtExp]) {
#pragma unroll
  for (int j = 0; j < kRtTok; ++j)
    xv[j] = (t0 + j < B) ? __ldg(xbase + (size_t)(t0 + j) * d4 + c4) : make_uint2(0u, 0u);
#pragma unroll
  for (int e = 0; e < kRtExp; ++e)
    wv[e] = (e0 + e < N) ? __ldg(wbase + (size_t)(e0 + e) * d4 + c4)
                         : make_float4(0.f, 0.f, 0.f, 0.f);
}

__global__ void __launch_bounds__(kRtWarps * 32) router_logits_kernel(
    const uint16_t *__restrict__ x, const float *__restrict__ Wg, float *__restrict__ h, int B,
    int N, int d) {
  __shared__ float red[kRtWarps][kRtOut];
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int e0 = blockIdx.x * kRtExp, t0 = blockIdx.y * kRtTok;
  const int d4 = d / 4;
  const int c_end = (warp + 1) * (d4 / kRtWarps);
  float acc[kRtOut];
#pragma unroll
  for (int i = 0; i < kRtOut; ++i) acc[i] = 0.f;
  const float4 *wbase = reinterpret_cast<const float4 *>(Wg);
  const uint2 *xbase = reinterpret_cast<const uint2 *>(x);
  int c4 = warp * (d4 / kRtWarps) + lane;
  uint2 xv[kRtTok];
  float4 wv[kRtExp];
  if (c4 < c_end) rt_load(xbase, wbase, t0, e0, B, N, d4, c4, xv, wv);
  while (c4 < c_end) {
    uint2 xn[kRtTok];
    float4 wn[kRtExp];
    const int cn = c4 + 32;
    if (cn < c_end) rt_load(xbase, wbase, t0, e0, B, N, d4, cn, xn, wn);
#pragma unroll
    for (int j = 0; j < kRtTok; ++j) {
      const float x0 = __uint_as_float(xv[j].x << 16), x1 = __uint_as_float(xv[j].x & 0xffff0000u);
      const float x2 = __uint_as_float(xv[j].y << 16), x3 = __uint_as_float(xv[j].y & 0xffff0000u);
#pragma unroll
      for (int e = 0; e < kRtExp; ++e) {
        float a = acc[j * kRtExp + e];
        a = fmaf(x0, wv[e].x, a);
        a = fmaf(x1, wv[e].y, a);
        a = fmaf(x2, wv[e].z, a);
        a = fmaf(x3, wv[e].w, a);
        acc[j * kRtExp + e] = a;
      }
    }
    if (cn < c_end) {
#pragma unroll
      for (int j = 0; j < kRtTok; ++j) xv[j] = xn[j];
#pragma unroll
      for (int e = 0; e < kRtExp; ++e) wv[e] = wn[e];
    }
    c4 = cn;
  }
  // Reduce-scatter: after the step with offset o a lane keeps the half of its
  // values selected by bit o of its lane id; after five steps lane l holds
  // the complete sum of output l.
#pragma unroll
  for (int o = 16, n = kRtOut / 2; o >= 1; o >>= 1, n >>= 1) {
    const bool upper = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < n; ++i) {
      const float lo = acc[i], hi = acc[i + n];
      const float recv = __shfl_xor_sync(kFull, upper ? lo : hi, o);
      acc[i] = (upper ? hi : lo) + recv;
    }
  }
  red[warp][lane] = acc[0];
  __syncthreads();
  if (threadIdx.x < kRtOut) {
    float sum = red[0][threadIdx.x];
#pragma unroll
    for (int w = 1; w < kRtWarps; ++w) sum += red[w][threadIdx.x];
    const int t = t0 + threadIdx.x / kRtExp, e = e0 + threadIdx.x % kRtExp;
    if (t < B && e < N) h[(size_t)t * N + e] = sum;
  }
}

// Xp[row] = x[token of pair perm[row]], 16-byte vectors.
__global__ void __launch_bounds__(256) gather_kernel(const uint16_t *__restrict__ x,
                                                     const int32_t *__restrict__ perm,
                                                     const Meta *__restrict__ meta,
                                                     uint16_t *__restrict__ xp, int d, int k) {
  pdl_wait();
  pdl_trigger();
  const int row = blockIdx.x;
  if (row >= meta->n_pairs) return;
  const int t = perm[row] / k;
  const uint4 *src = reinterpret_cast<const uint4 *>(x + (size_t)t * d);
  uint4 *dst = reinterpret_cast<uint4 *>(xp + (size_t)row * d);
  for (int i = threadIdx.x; i < d / 8; i += blockDim.x) dst[i] = __ldg(src + i);
}

// ---- a9: y_t = sum over slots s < k' of w_ts * out[pos(t, s)], fp32, bf16 once.
__global__ void __launch_bounds__(256) combine_kernel(const float *__restrict__ out,
                                                      const int32_t *__restrict__ pos,
                                                      const float *__restrict__ w,
                                                      const Meta *__restrict__ meta,
                                                      uint16_t *__restrict__ y, int d, int k) {
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.y;
  const int c4 = blockIdx.x * blockDim.x + threadIdx.x;
  if (c4 >= d / 4) return;
  const int kp = meta->kprime;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int s = 0; s < kp; ++s) {
    const int r = pos[(size_t)t * k + s];
    if (r < 0) continue;  // only with non-finite scores
    const float ws = w[(size_t)t * k + s];
    const float4 o = reinterpret_cast<const float4 *>(out + (size_t)r * d)[c4];
    acc.x = fmaf(ws, o.x, acc.x);
    acc.y = fmaf(ws, o.y, acc.y);
    acc.z = fmaf(ws, o.z, acc.z);
    acc.w = fmaf(ws, o.w, acc.w);
  }
  __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x, acc.y);
  __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z, acc.w);
  uint2 v;
  v.x = *reinterpret_cast<uint32_t *>(&lo);
  v.y = *reinterpret_cast<uint32_t *>(&hi);
  reinterpret_cast<uint2 *>(y + (size_t)t * d)[c4] = v;
}

}  // namespace

size_t route_dynamic_smem(int B, int N, int k, bool *p_smem, bool *ids_smem) {
  const size_t p_bytes = (size_t)B * N * 4, ids_bytes = (size_t)B * k * 4;
  *p_smem = p_bytes <= kRouteSmemP;
  *ids_smem = ids_bytes <= kRouteSmemIds;
  const size_t wcnt_bytes = N <= kScatterMaxN ? (size_t)32 * N * 4 : 0;
  return (*p_smem ? p_bytes : 0) + (*ids_smem ? ids_bytes : 0) + wcnt_bytes;
}

template <int kMaxQ>
cudaError_t launch_route_q(RouteArgs a, cudaStream_t s) {
  bool ps = false, is = false;
  const size_t dyn = route_dynamic_smem(a.B, a.N, a.k, &ps, &is);
  a.p_smem = ps ? 1 : 0;
  a.ids_smem = is ? 1 : 0;
  cudaError_t e = cudaFuncSetAttribute(route_kernel<kMaxQ>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  if (e != cudaSuccess) return e;
  return launch_pdl(route_kernel<kMaxQ>, dim3(1), dim3(kRouteThreads), dyn, s, a);
}

cudaError_t launch_route(const RouteArgs &a, cudaStream_t s) {
  if (a.N <= 64) return launch_route_q<2>(a, s);
  if (a.N <= 128) return launch_route_q<4>(a, s);
  if (a.N <= 256) return launch_route_q<8>(a, s);
  return launch_route_q<32>(a, s);
}

cudaError_t launch_router_logits(const uint16_t *x, const float *Wg, float *h, int B, int N,
                                 int d, cudaStream_t s) {
  dim3 grid((N + kRtExp - 1) / kRtExp, (B + kRtTok - 1) / kRtTok);
  return launch_pdl(router_logits_kernel, grid, dim3(kRtWarps * 32), 0, s, x, Wg, h, B, N, d);
}

cudaError_t launch_gather(const uint16_t *x, const int32_t *perm, const Meta *meta,
                          uint16_t *xp, int max_pairs, int d, int k, cudaStream_t s) {
  return launch_pdl(gather_kernel, dim3(max_pairs), dim3(256), 0, s, x, perm, meta, xp, d, k);
}

cudaError_t launch_combine(const float *out, const int32_t *pos, const float *w,
                           const Meta *meta, uint16_t *y, int B, int d, int k,
                           cudaStream_t s) {
  dim3 grid((d / 4 + 255) / 256, B);
  return launch_pdl(combine_kernel, grid, dim3(256), 0, s, out, pos, w, meta, y, d, k);
}

}  // namespace xs
