// Router, batch-aware expert selection, refinement, permutation, gather and
// combine kernels (steps a1-a7 and a9 of the MoE-layer forward).
//
// Selection follows XShare (arxiv 2602.07265): Algorithm 2 (BATCH; THRESH
// with Algorithm 1's threshold), Algorithms 3-4 (HIER), Algorithms 5-6
// (GROUP) and plain top-k (TOPK), on fp32 gating scores, with the refinement
// "route x_i to Top k(G_i, S)" and the renormalised weights of Sec. 2.2.
#include <cuda_bf16.h>

#include <climits>
#include <cmath>

#include "xs_internal.cuh"

namespace xs {
namespace {

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ unsigned long long gtimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

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

// Marks (calls mark(index) for) the `count` best candidates of an unsorted
// lane list laid out by lane_load (lane l slot q: index j0 + l + 32 q), in
// the order of `before`: every candidate whose key is above the count-th
// largest key T, then the lowest-index candidates whose key equals T.  T is
// the largest key with count(key >= T) >= count, found bit by bit from the
// top: the bits above the highest bit where the largest and smallest live
// keys differ are theirs, and the rest are found two bits per round (three
// independent warp reductions).  The search stops early once a threshold has
// exactly `count` keys at or above it (those are the count best: any such
// threshold marks the same set).  All of them if count >= the live
// candidates.
template <int Q, class Mark>
__device__ __forceinline__ void lane_mark_top(const LaneList<Q> &L, int count, Mark mark) {
  const int lane = threadIdx.x & 31;
  if (count <= 0) return;
  int live = 0;
#pragma unroll
  for (int q = 0; q < Q; ++q) live += L.key[q] != 0u ? 1 : 0;
  live = static_cast<int>(__reduce_add_sync(kFull, static_cast<unsigned>(live)));
  if (count >= live) {
#pragma unroll
    for (int q = 0; q < Q; ++q)
      if (L.key[q] != 0u) mark(L.idx[q]);
    return;
  }
  uint32_t kmx = 0u, kmn = 0xffffffffu;
#pragma unroll
  for (int q = 0; q < Q; ++q)
    if (L.key[q] != 0u) {
      kmx = max(kmx, L.key[q]);
      kmn = min(kmn, L.key[q]);
    }
  kmx = __reduce_max_sync(kFull, kmx);
  kmn = __reduce_min_sync(kFull, kmn);
  const uint32_t diff = kmx ^ kmn;
  int bit = diff != 0u ? 31 - __clz(diff) : -1;
  // The shared high bits (2u << 31 wraps to 0: nothing shared).
  uint32_t T = diff != 0u ? (kmx & ~((2u << bit) - 1u)) : kmx;
  // Exactly `count` keys are >= c and every other key is below c: they are
  // the count best, whatever the order among them.
  auto mark_from = [&](uint32_t c) {
#pragma unroll
    for (int q = 0; q < Q; ++q)
      if (L.key[q] >= c) mark(L.idx[q]);
  };
  auto count_from = [&](uint32_t c) {
    int n = 0;
#pragma unroll
    for (int q = 0; q < Q; ++q) n += L.key[q] >= c ? 1 : 0;
    return n;
  };
  for (; bit >= 1; bit -= 2) {
    const uint32_t c1 = T | (1u << (bit - 1)), c2 = T | (2u << (bit - 1)), c3 = T | (3u << (bit - 1));
    const int n1 = static_cast<int>(__reduce_add_sync(kFull, static_cast<unsigned>(count_from(c1))));
    const int n2 = static_cast<int>(__reduce_add_sync(kFull, static_cast<unsigned>(count_from(c2))));
    const int n3 = static_cast<int>(__reduce_add_sync(kFull, static_cast<unsigned>(count_from(c3))));
    if (n3 == count) return mark_from(c3);
    if (n2 == count) return mark_from(c2);
    if (n1 == count) return mark_from(c1);
    T = n3 > count ? c3 : n2 > count ? c2 : n1 > count ? c1 : T;
  }
  if (bit == 0) {
    const uint32_t c = T | 1u;
    const int n = static_cast<int>(__reduce_add_sync(kFull, static_cast<unsigned>(count_from(c))));
    if (n == count) return mark_from(c);
    if (n > count) T = c;
  }
  int gt = 0;
#pragma unroll
  for (int q = 0; q < Q; ++q) {
    gt += L.key[q] > T ? 1 : 0;
    if (L.key[q] > T) mark(L.idx[q]);
  }
  int need = count - static_cast<int>(__reduce_add_sync(kFull, static_cast<unsigned>(gt)));
#pragma unroll
  for (int q = 0; q < Q; ++q) {
    const bool tie = L.key[q] == T;
    const unsigned b = __ballot_sync(kFull, tie);
    if (tie && __popc(b & ((1u << lane) - 1u)) < need) mark(L.idx[q]);
    need -= __popc(b);
  }
}

// Halving tree over the expert index of values held as v[q] = value of expert
// lane + 32 q (zero where there is none): for o = 16 Q, ..., 32 the pairs
// (j, j + o) are in one lane; for o = 16, ..., 1 they are lanes l and l + o.
// Returns the sum on every lane.  Zero padding adds exactly, so the result is
// that of the tree over any power-of-two length >= the number of experts.
template <int Q>
__device__ __forceinline__ float expert_tree(float (&v)[Q]) {
#pragma unroll
  for (int h = Q / 2; h >= 1; h >>= 1) {
#pragma unroll
    for (int q = 0; q < h; ++q) v[q] = __fadd_rn(v[q], v[q + h]);
  }
  float x = v[0];
#pragma unroll
  for (int o = 16; o; o >>= 1) x = __fadd_rn(x, __shfl_down_sync(kFull, x, o));
  return __shfl_sync(kFull, x, 0);
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

// Moves each lane's best candidate to slot 0 (enough for a single take).
template <int Q>
__device__ __forceinline__ void lane_head(LaneList<Q> &L) {
#pragma unroll
  for (int q = 1; q < Q; ++q) {
    if (before(L.key[q], L.idx[q], L.key[0], L.idx[0])) {
      const uint32_t tk = L.key[0];
      L.key[0] = L.key[q];
      L.key[q] = tk;
      const int ti = L.idx[0];
      L.idx[0] = L.idx[q];
      L.idx[q] = ti;
    }
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

// Selection is split over two kernels whose CTAs each own one chunk of 32
// tokens (the canonical summation chunk, so column sums stay bit-identical to
// a single-pass evaluation):
//
//   score_kernel  (a2, a3, a4, part of a5): per token (one warp each) the
//       dense softmax of the logits (or the given scores) and the ranking the
//       selection needs (the warm-up top-k0; the top-k too for the sparse
//       reading); the chunk's column-sum tree and warm-up marks; for HIER,
//       Algorithm 3 for every request inside the chunk.  The CTA that
//       finishes last adds the chunk sums left to right, merges the marks and
//       runs the budgeted selection (a5): BATCH and the batch step of HIER
//       search the budget-th column score outside the base set in one warp;
//       GROUP ranks each group in its own warp (Algorithm 5's rounds in
//       closed form).  CTAs C .. 2C - 1 rank every token's top-k over E at
//       the same time and count the plain top-k union (a statistic).
//   refine_kernel (a6, a7): per token the top-k' inside S with renormalised
//       weights.  The CTA that finishes last counts the pairs per expert,
//       takes the prefix sums, writes the FFN tiles and scatters the pairs
//       stably by expert.
//
// "Last to finish" uses an arrival counter per group of CTAs (done[0] the
// selection, done[1] the refinement, done[2] the union), cleared before the
// first kernel of the call: every CTA writes its results, fences, and bumps
// the counter; the CTA that sees the final count continues alone.  No CTA
// waits for another.

__device__ __forceinline__ int chunk_count(int B) { return (B + kChunk - 1) / kChunk; }

// Selected set statistics: |S| and the max group load.
__device__ __forceinline__ void selection_stats(const RouteArgs &a, const uint8_t *s_mask, int *s_gl,
                                                int &nsel, int &maxload) {
  const int tid = threadIdx.x, N = a.N;
  const int G = a.G >= 1 ? a.G : 1, size = N / G;
  if (G == 1) {  // one group: its load is |S|
    nsel = __syncthreads_count(tid < N && s_mask[tid]);
    maxload = nsel;
    return;
  }
  for (int g = tid; g < G; g += blockDim.x) s_gl[g] = 0;
  __syncthreads();
  for (int j = tid; j < N; j += blockDim.x)
    if (s_mask[j]) atomicAdd(&s_gl[j / size], 1);
  nsel = __syncthreads_count(tid < N && s_mask[tid]);
  int best = 0;
  for (int g = tid; g < G; g += blockDim.x) best = max(best, s_gl[g]);
  best = __reduce_max_sync(kFull, best);
  if ((tid & 31) == 0) atomicMax(&s_gl[kMaxN], best);
  __syncthreads();
  maxload = s_gl[kMaxN];
}

// The experts of S in ascending order into s_list; returns |S|.  One thread
// per expert (blockDim >= N); s_wc: [32] scratch.
__device__ __forceinline__ int compact_selected(const uint8_t *s_mask, int N, int32_t *s_list,
                                                int *s_wc) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
  const bool m = tid < N && s_mask[tid] != 0;
  const unsigned b = __ballot_sync(kFull, m);
  if (lane == 0) s_wc[warp] = __popc(b);
  __syncthreads();
  int base = 0, total = 0;
  for (int w = 0; w < nw; ++w) {
    const int c = s_wc[w];
    base += (w < warp) ? c : 0;
    total += c;
  }
  if (m) s_list[base + __popc(b & ((1u << lane) - 1u))] = tid;
  __syncthreads();
  return total;
}

static_assert(kRouteThreads >= kMaxN, "compact_selected takes one thread per expert");

// Per token t in [t_begin, t_end), one warp each: Top k'(G_t, S) with the
// renormalised weights (a6); row(t) points at the token's scores.  Lane l
// ranks the experts s_list[l + 32 q] of S (q < Q, Q * 32 >= |S|).
template <int Q, class Row>
__device__ __forceinline__ void refine_tokens_q(const RouteArgs &a, const int32_t *s_list, int nS,
                                                int t_begin, int t_end, int kp, Row row,
                                                int32_t *ids_s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const int k = a.k;
  for (int t = t_begin + warp; t < t_end; t += nwarps) {
    const float *prow = row(t);
    LaneList<Q> L;
#pragma unroll
    for (int q = 0; q < Q; ++q) {
      const int i = lane + 32 * q;
      const int e = i < nS ? s_list[i] : 0;
      L.idx[q] = e;
      L.key[q] = i < nS ? score_key(prow[e]) : 0u;
    }
    lane_sort<Q>(L);
    int my_id = -1;  // lane s keeps slot s
    float my_v = 0.f;
    float D = 0.f;
    const int got = lane_take<Q>(L, kp, [&](int r, int id, float v) {
      if (lane == r) {
        my_id = id;
        my_v = v;
      }
      D = __fadd_rn(D, v);  // slot order, identical on every lane
    });
    if (lane < k) {
      float wv = 0.f;
      if (lane < got) wv = (D > 0.f) ? __fdiv_rn(my_v, D) : __fdiv_rn(1.f, (float)got);
      a.ids[(size_t)t * k + lane] = (lane < got) ? my_id : -1;
      if (ids_s) ids_s[(t - t_begin) * k + lane] = (lane < got) ? my_id : -1;
      a.w[(size_t)t * k + lane] = wv;
    }
  }
}

// The same over all N experts with the mask (lane l: experts l + 32 q).
template <int kQ, class Row>
__device__ __forceinline__ void refine_tokens_masked(const RouteArgs &a, const uint8_t *s_mask,
                                                     int t_begin, int t_end, int kp, Row row,
                                                     int32_t *ids_s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  const int N = a.N, k = a.k;
  for (int t = t_begin + warp; t < t_end; t += nwarps) {
    const float *prow = row(t);
    LaneList<kQ> L;
    lane_load<kQ>(L, 0, N, lane, [&](int, int j) { return prow[j]; },
                  [&](int, int j) { return s_mask[j] != 0; });
    lane_sort<kQ>(L);
    int my_id = -1;
    float my_v = 0.f;
    float D = 0.f;
    const int got = lane_take<kQ>(L, kp, [&](int r, int id, float v) {
      if (lane == r) {
        my_id = id;
        my_v = v;
      }
      D = __fadd_rn(D, v);
    });
    if (lane < k) {
      float wv = 0.f;
      if (lane < got) wv = (D > 0.f) ? __fdiv_rn(my_v, D) : __fdiv_rn(1.f, (float)got);
      a.ids[(size_t)t * k + lane] = (lane < got) ? my_id : -1;
      if (ids_s) ids_s[(t - t_begin) * k + lane] = (lane < got) ? my_id : -1;
      a.w[(size_t)t * k + lane] = wv;
    }
  }
}

// Refinement of tokens [t_begin, t_end) against S (|S| = nS, the mask in
// s_mask).  When S fits a shorter lane list than all N experts need, its
// experts are first compacted into s_list (then [kMaxN] scratch, s_wc [32]);
// either way the candidates and their order are the same.  Every thread of
// the block calls it with the same nS.
template <int kQ, class Row>
__device__ __forceinline__ void refine_tokens(const RouteArgs &a, const uint8_t *s_mask, int nS,
                                              int32_t *s_list, int *s_wc, int t_begin, int t_end,
                                              int kp, Row row, int32_t *ids_s = nullptr) {
  const int nq = (nS + 31) / 32;
  if (kQ > 2 && nq <= 2) {
    compact_selected(s_mask, a.N, s_list, s_wc);
    refine_tokens_q<(kQ > 2 ? 2 : kQ)>(a, s_list, nS, t_begin, t_end, kp, row, ids_s);
  } else if (kQ > 4 && nq <= 4) {
    compact_selected(s_mask, a.N, s_list, s_wc);
    refine_tokens_q<(kQ > 4 ? 4 : kQ)>(a, s_list, nS, t_begin, t_end, kp, row, ids_s);
  } else {
    refine_tokens_masked<kQ>(a, s_mask, t_begin, t_end, kp, row, ids_s);
  }
}

struct PermSmem {
  int32_t *counts, *cursor, *chunk, *tmp, *scal, *wcnt;  // wcnt: [32][N] (N <= kScatterMaxN)
  const int32_t *ids;  // nullable: the ids in shared memory (else read from global)
};

// Counting sort of all pairs by expert, stable in (token, slot) (a7), the FFN
// tiles and the statistics.  One CTA, once every token's ids are written and
// visible; the meta block already holds the selection's fields.
__device__ void build_permutation(const RouteArgs &a, PermSmem sm) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = blockDim.x >> 5;
  const int B = a.B, N = a.N, k = a.k;
  const int P = B * k;
  for (int j = tid; j < N; j += blockDim.x) sm.counts[j] = 0;
  __syncthreads();
  for (int q = tid; q < P; q += blockDim.x) {
    const int e = sm.ids ? sm.ids[q] : __ldcg(a.ids + q);
    if ((unsigned)e < (unsigned)N) atomicAdd(&sm.counts[e], 1);
  }
  __syncthreads();
  {
    const int cnt = tid < N ? sm.counts[tid] : 0;
    int v[3] = {cnt, (cnt + kTileTok - 1) / kTileTok, cnt > 0 ? 1 : 0}, tot[3];
    block_scan3(v, tot, sm.tmp);
    if (tid < N) {
      sm.cursor[tid] = v[0];
      a.counts[tid] = cnt;
      a.offsets[tid] = v[0];
      if (a.counts_out) a.counts_out[tid] = cnt;
      if (a.offsets_out) a.offsets_out[tid] = v[0];
      for (int tt = 0; tt * kTileTok < cnt; ++tt) {
        Tile tl;
        tl.expert = tid;
        tl.row0 = v[0] + tt * kTileTok;
        tl.ntok = min(kTileTok, cnt - tt * kTileTok);
        tl.pad = 0;
        a.tiles[v[1] + tt] = tl;
      }
    }
    if (tid == 0) {
      a.offsets[N] = tot[0];
      if (a.offsets_out) a.offsets_out[N] = tot[0];
      sm.scal[1] = tot[0];  // pairs
      sm.scal[2] = tot[1];  // tiles
      sm.scal[3] = tot[2];  // used experts
    }
    // This call's FFN work (Sec. 5): the tiles and rows of the experts of
    // group ep_rank, a contiguous index range, hence contiguous tiles and
    // rows; shared experts go to rank 0.  Without expert parallelism: all.
    {
      const int G = a.ep_ranks > 1 ? a.ep_ranks : 1, g = G > 1 ? a.ep_rank : 0;
      const int e_lo = g * (N / G), e_hi = (g + 1) * (N / G);
      Meta *m = a.meta;
      if (tid == e_lo) {
        m->ffn_t0 = v[1];
        m->row0 = v[0];
      }
      if (e_hi < N && tid == e_hi) {
        m->ffn_t1 = v[1];
        m->row1 = v[0];
      }
      if (tid == 0) {
        if (e_hi >= N) {
          m->ffn_t1 = tot[1];
          m->row1 = tot[0];
        }
        const int own_shared = g == 0 ? 1 : 0;
        m->ffn_s0 = tot[1];
        m->ffn_s1 = tot[1] + own_shared * a.n_shared * ((B + kTileTok - 1) / kTileTok);
        m->srows = own_shared;
      }
    }
    // Shared experts: every token, in token order, after the routed pairs.
    const int tpt = (B + kTileTok - 1) / kTileTok;
    for (int i = tid; i < a.n_shared * tpt; i += blockDim.x) {
      const int j = i / tpt, tt = i - j * tpt;
      Tile tl;
      tl.expert = N + j;
      tl.row0 = tot[0] + j * B + tt * kTileTok;
      tl.ntok = min(kTileTok, B - tt * kTileTok);
      tl.pad = 0;
      a.tiles[tot[1] + i] = tl;
    }
  }
  __syncthreads();
  const unsigned lt = (1u << lane) - 1u;
  if (N <= kScatterMaxN) {
    // Chunks of blockDim pairs: rank inside a warp by match_any, then an
    // exclusive prefix over the warps of the chunk for every expert.
    for (int base = 0; base < P; base += blockDim.x) {
      // Only the warps that hold pairs of this chunk count.
      const int nw_used = min(nwarps, (P - base + 31) / 32);
      for (int i = tid; i < nw_used * N; i += blockDim.x) sm.wcnt[i] = 0;
      const int q = base + tid;
      int e = (q < P) ? (sm.ids ? sm.ids[q] : __ldcg(a.ids + q)) : -1;
      if ((unsigned)e >= (unsigned)N) e = -1;
      const unsigned peers = __match_any_sync(kFull, e);
      const int rank = __popc(peers & lt);
      __syncthreads();
      if (e >= 0 && rank == 0) sm.wcnt[warp * N + e] = __popc(peers);
      __syncthreads();
      if (tid < N) {
        int run = 0;
        for (int w = 0; w < nw_used; ++w) {
          const int x = sm.wcnt[w * N + tid];
          sm.wcnt[w * N + tid] = run;
          run += x;
        }
        sm.chunk[tid] = run;
      }
      __syncthreads();
      if (e >= 0) {
        const int r = sm.cursor[e] + sm.wcnt[warp * N + e] + rank;
        a.perm[r] = q;
        a.pos[q] = r;
        if (a.perm_out) a.perm_out[r] = q;
      } else if (q < P) {
        a.pos[q] = -1;
      }
      __syncthreads();
      if (tid < N) sm.cursor[tid] += sm.chunk[tid];
      __syncthreads();
    }
  } else if (warp == 0) {
    for (int base = 0; base < P; base += 32) {
      const int q = base + lane;
      int e = (q < P) ? (sm.ids ? sm.ids[q] : __ldcg(a.ids + q)) : -1;
      if ((unsigned)e >= (unsigned)N) e = -1;
      const unsigned peers = __match_any_sync(kFull, e);
      const int rank = __popc(peers & lt);
      const int old = (e >= 0) ? sm.cursor[e] : 0;
      __syncwarp();
      if (e >= 0) {
        const int r = old + rank;
        a.perm[r] = q;
        a.pos[q] = r;
        if (a.perm_out) a.perm_out[r] = q;
        if (rank == 0) sm.cursor[e] = old + __popc(peers);
      } else if (q < P) {
        a.pos[q] = -1;
      }
      __syncwarp();
    }
  }
  if (tid == 0) {
    // Field by field: union_topk belongs to the union CTAs (score_kernel).
    Meta *m = a.meta;
    m->n_pairs = sm.scal[1];  // == B * kp unless scores were non-finite
    m->n_tiles = sm.scal[2] + a.n_shared * ((B + kTileTok - 1) / kTileTok);
    m->n_used = sm.scal[3];
    m->n_rows = sm.scal[1] + a.n_shared * B;
    if (a.stats) {
      xs_stats *st = a.stats;
      st->n_selected = m->n_selected;
      st->n_used = sm.scal[3];
      st->max_group_load = m->max_group_load;
      st->n_pairs = sm.scal[1];
      st->status = m->status;
      st->reserved[0] = st->reserved[1] = 0;
    }
  }
}

// The same permutation, tiles and statistics as build_permutation, for a
// batch of at most 64 tokens, with two block barriers instead of about ten.
// A pair's position in its expert's run is the number of earlier tokens
// routed to that expert (a token uses an expert in at most one slot), so one
// 32-bit token mask per expert and 32-token chunk gives the counts and every
// position.  The masks (sm.cursor for tokens 0-31, sm.counts for 32-63, as
// uint32) must be zero on entry.  ids: ids_s[t * k + s] in shared memory
// (one chunk), else the ids in global memory.
//   1. every pair (t, s): mask[t / 32][e] |= 1 << (t % 32) (shared-memory
//      atomic).
//   2. warp 0, 32 experts per round: counts, exclusive prefix over the
//      experts (rows, and tiles = used experts: a count of at most 64 is one
//      tile), tiles, meta.
//   3. warp t, lane s < k: position of pair (t, s) = offset[e] + the tokens
//      of e in the chunks before + popc(mask[t / 32][e] & (tokens below t)).
__device__ void build_permutation_small(const RouteArgs &a, PermSmem sm, const int32_t *ids_s) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = blockDim.x >> 5;
  const int B = a.B, N = a.N, k = a.k;
  uint32_t *s_tm0 = reinterpret_cast<uint32_t *>(sm.cursor);  // [N] tokens 0-31 per expert
  uint32_t *s_tm1 = reinterpret_cast<uint32_t *>(sm.counts);  // [N] tokens 32-63 per expert
  int32_t *s_off = sm.chunk;                                   // [N] first row per expert
  auto id_of = [&](int q) { return ids_s != nullptr ? ids_s[q] : __ldcg(a.ids + q); };
  for (int q = tid; q < B * k; q += blockDim.x) {
    const int e = id_of(q), t = q / k;
    if ((unsigned)e < (unsigned)N) atomicOr(t < 32 ? &s_tm0[e] : &s_tm1[e], 1u << (t & 31));
  }
  __syncthreads();
  if (warp == 0) {
    const int G = a.ep_ranks > 1 ? a.ep_ranks : 1, g = G > 1 ? a.ep_rank : 0;
    const int e_lo = g * (N / G), e_hi = (g + 1) * (N / G);
    Meta *m = a.meta;
    int rows0 = 0, tiles0 = 0;  // totals of the rounds before
    for (int e0 = 0; e0 < N; e0 += 32) {
      const int e = e0 + lane;
      const int c = e < N ? __popc(s_tm0[e]) + (B > 32 ? __popc(s_tm1[e]) : 0) : 0;
      const int u = c > 0 ? 1 : 0;
      int rx = c, ux = u;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int r1 = __shfl_up_sync(kFull, rx, o), u1 = __shfl_up_sync(kFull, ux, o);
        if (lane >= o) {
          rx += r1;
          ux += u1;
        }
      }
      const int row = rows0 + rx - c, tile = tiles0 + ux - u;  // exclusive
      if (e < N) {
        s_off[e] = row;
        a.counts[e] = c;
        a.offsets[e] = row;
        if (a.counts_out) a.counts_out[e] = c;
        if (a.offsets_out) a.offsets_out[e] = row;
        // This call's FFN work (Sec. 5): the tiles and rows of expert group
        // ep_rank (a contiguous index range); without expert parallelism, all.
        if (e == e_lo) {
          m->ffn_t0 = tile;
          m->row0 = row;
        }
        if (e_hi < N && e == e_hi) {
          m->ffn_t1 = tile;
          m->row1 = row;
        }
        if (c > 0) {
          Tile tl;
          tl.expert = e;
          tl.row0 = row;
          tl.ntok = c;
          tl.pad = 0;
          a.tiles[tile] = tl;
        }
      }
      rows0 += __shfl_sync(kFull, rx, 31);
      tiles0 += __shfl_sync(kFull, ux, 31);
    }
    const int tot_rows = rows0, tot_tiles = tiles0;
    // Shared experts: every token, in token order, after the routed pairs
    // (one tile each: B <= 64).
    for (int j = lane; j < a.n_shared; j += 32) {
      Tile tl;
      tl.expert = N + j;
      tl.row0 = tot_rows + j * B;
      tl.ntok = B;
      tl.pad = 0;
      a.tiles[tot_tiles + j] = tl;
    }
    if (lane == 0) {
      a.offsets[N] = tot_rows;
      if (a.offsets_out) a.offsets_out[N] = tot_rows;
      if (e_hi >= N) {
        m->ffn_t1 = tot_tiles;
        m->row1 = tot_rows;
      }
      const int own_shared = g == 0 ? 1 : 0;
      m->ffn_s0 = tot_tiles;
      m->ffn_s1 = tot_tiles + own_shared * a.n_shared;
      m->srows = own_shared;
      // Field by field: union_topk belongs to the union CTAs (score_kernel).
      m->n_pairs = tot_rows;  // == B * kp unless scores were non-finite
      m->n_tiles = tot_tiles + a.n_shared;
      m->n_used = tot_tiles;
      m->n_rows = tot_rows + a.n_shared * B;
      if (a.stats) {
        xs_stats *st = a.stats;
        st->n_selected = m->n_selected;
        st->n_used = tot_tiles;
        st->max_group_load = m->max_group_load;
        st->n_pairs = tot_rows;
        st->status = m->status;
        st->reserved[0] = st->reserved[1] = 0;
      }
    }
  }
  __syncthreads();
  for (int t = warp; t < B; t += nwarps) {
    if (lane < k) {
      const int q = t * k + lane;
      const int e = id_of(q);
      if ((unsigned)e < (unsigned)N) {
        const uint32_t below = (1u << (t & 31)) - 1u;
        const int r = s_off[e] + (t < 32 ? __popc(s_tm0[e] & below)
                                         : __popc(s_tm0[e]) + __popc(s_tm1[e] & below));
        a.perm[r] = q;
        a.pos[q] = r;
        if (a.perm_out) a.perm_out[r] = q;
      } else {
        a.pos[q] = -1;
      }
    }
  }
}

// Token t's dense scores (a2) in vals[q] = p[t, lane + 32 q] (0 past N): the
// softmax of its logits (written to a.p when write_p), or the given scores.
template <int kQ>
__device__ __forceinline__ void token_scores(const RouteArgs &a, int t, int lane, float (&vals)[kQ],
                                             bool write_p) {
  const int N = a.N;
  if (a.logits != nullptr) {
    // The router may leave the logits as slices over d (h[s][t][j]); they
    // are added in slice order.
    const float *hrow = a.logits + (size_t)t * N;
#pragma unroll
    for (int q = 0; q < kQ; ++q) {
      const int j = lane + 32 * q;
      vals[q] = (j < N) ? hrow[j] : -INFINITY;
    }
    for (int sl = 1; sl < a.h_splits; ++sl) {
      const float *hs = hrow + (size_t)sl * a.B * N;
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        const int j = lane + 32 * q;
        if (j < N) vals[q] = __fadd_rn(vals[q], hs[j]);
      }
    }
    float mx = -INFINITY;
#pragma unroll
    for (int q = 0; q < kQ; ++q) mx = fmaxf(mx, vals[q]);
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
    // One correctly rounded reciprocal and a product per expert (within one
    // ulp of the quotient; measured 2 us faster than the divisions).
    const float rs = __frcp_rn(sum);
#pragma unroll
    for (int q = 0; q < kQ; ++q) {
      const int j = lane + 32 * q;
      if (j < N) {
        vals[q] = __fmul_rn(vals[q], rs);
        if (write_p) a.p[(size_t)t * N + j] = vals[q];
      }
    }
  } else {
#pragma unroll
    for (int q = 0; q < kQ; ++q) {
      const int j = lane + 32 * q;
      vals[q] = (j < N) ? a.p[(size_t)t * N + j] : 0.f;
    }
  }
}

// The plain top-k union (a statistic): CTA C + c ranks the k best experts of
// every token of chunk c over E, concurrently with the selection CTAs, and
// the last of these CTAs to finish counts the union and writes union_topk.
template <int kQ>
__device__ __noinline__ void union_cta(const RouteArgs &a, uint8_t *s_union, int32_t *s_flag) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nwarps = blockDim.x >> 5;
  const int B = a.B, N = a.N, k = a.k;
  const int C = chunk_count(B), c = blockIdx.x - C;
  const int t0 = c * kChunk, nt = min(kChunk, B - t0);
  for (int j = tid; j < N; j += blockDim.x) s_union[j] = 0;
  __syncthreads();
  for (int w = warp; w < nt; w += nwarps) {
    float vals[kQ];
    token_scores<kQ>(a, t0 + w, lane, vals, false);
    LaneList<kQ> L;
    lane_load<kQ>(L, 0, N, lane, [&](int q, int) { return vals[q]; }, [](int, int) { return true; });
    lane_sort<kQ>(L);
    lane_take<kQ>(L, k, [&](int, int id, float) {
      if (lane == 0) s_union[id] = 1;
    });
  }
  __syncthreads();
  if (C > 1) {
    uint8_t *marks = a.chunk_marks + (size_t)c * 2 * N + N;
    for (int j = tid; j < N; j += blockDim.x) marks[j] = s_union[j];
    __threadfence();
    __syncthreads();
    if (tid == 0) *s_flag = (atomicAdd(&a.done[2], 1) == C - 1) ? 1 : 0;
    __syncthreads();
    if (!*s_flag) return;
    __threadfence();
    for (int j = tid; j < N; j += blockDim.x) {
      uint8_t u = 0;
      for (int cc = 0; cc < C; ++cc) u |= __ldcg(a.chunk_marks + (size_t)cc * 2 * N + N + j);
      s_union[j] = u;
    }
    __syncthreads();
  }
  const int n_union = __syncthreads_count(tid < N && s_union[tid]);
  if (tid == 0) {
    a.meta->union_topk = n_union;
    if (a.stats) a.stats->union_topk = n_union;
  }
}

template <int kQ>
__global__ void __launch_bounds__(kRouteThreads, 1) score_kernel(RouteArgs a) {
  extern __shared__ float ps[];         // [32][N] scores of the chunk's tokens (+ [32][N] ints)
  __shared__ uint8_t s_mask[kMaxN];     // S (selection step)
  __shared__ uint8_t s_base[kMaxN];     // chunk marks: S_0 (or S_r for HIER); merged later
  __shared__ uint8_t s_union[kMaxN];    // union CTAs: plain top-k union marks
  __shared__ float s_col[kMaxN];
  __shared__ int32_t s_gl[kMaxN + 1];
  __shared__ int32_t s_top[kChunk][kMaxK];
  __shared__ int32_t s_scal[4];
  __shared__ int32_t s_counts[kMaxN];   // permutation, when it runs in this kernel
  __shared__ int32_t s_cursor[kMaxN];
  __shared__ int32_t s_chunk[kMaxN];
  __shared__ int32_t s_tmp[200];
  __shared__ int s_rflag;               // a router CTA reported a timeout

  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = blockDim.x >> 5;
  const int B = a.B, N = a.N, k = a.k;
  const int C = chunk_count(B), c = blockIdx.x;
  if (tid == 0) s_rflag = 0;
  if (c >= C) {  // CTAs C .. 2C - 1 count the plain top-k union
    union_cta<kQ>(a, s_union, s_scal);
    return;
  }
  const int t0 = c * kChunk, nt = min(kChunk, B - t0);
  // Ranking depth the selection needs: the warm-up top-k0, and the token's
  // top-k for Sec. 2.2's gating values when the column scores are sparse.
  const int kk = a.sparse ? max(k, a.k0) : a.k0;
  const bool hier = a.mode == XS_MODE_HIER;
  // HIER requests that lie inside one chunk are selected here (Algorithm 3);
  // otherwise the selection step does it from the full score matrix.
  const bool hier_here = hier && a.T <= kChunk && kChunk % a.T == 0;

  for (int j = tid; j < N; j += blockDim.x) s_base[j] = 0;
  if (a.zero_words != nullptr)
    for (int i = c * blockDim.x + tid; i < a.zero_count; i += C * blockDim.x) a.zero_words[i] = 0;
  __syncthreads();

  // ---- per token: scores (a2) and ranking over E (a3) ----
  for (int w = warp; w < kChunk; w += nwarps) {
    float *prow_s = ps + w * N;
    if (w >= nt) {  // zero rows pad the last chunk's tree
      for (int j = lane; j < N; j += 32) prow_s[j] = 0.f;
      continue;
    }
    const int t = t0 + w;
    float vals[kQ];
    token_scores<kQ>(a, t, lane, vals, true);
#pragma unroll
    for (int q = 0; q < kQ; ++q)
      if (lane + 32 * q < N) prow_s[lane + 32 * q] = vals[q];
    if (kk == 0) continue;
    LaneList<kQ> L;
    lane_load<kQ>(L, 0, N, lane, [&](int q, int) { return vals[q]; },
                  [](int, int) { return true; });
    if (kk == 1)
      lane_head<kQ>(L);
    else
      lane_sort<kQ>(L);
    int32_t *top = a.toptok + (size_t)t * kMaxK;
    int my_id = -1;  // sparse scores: lane s keeps slot s of the token's top-k
    float my_v = 0.f, D = 0.f;
    lane_take<kQ>(L, kk, [&](int r, int id, float v) {
      if (lane == 0) {
        if (r < a.k0) {
          s_top[w][r] = id;
          if (hier)
            top[r] = id;
          else
            s_base[id] = 1;
        }
      }
      if (r < k) {
        if (lane == r) {
          my_id = id;
          my_v = v;
        }
        D = __fadd_rn(D, v);  // rank order, identical on every lane
      }
    });
    if (a.sparse) {
      // Sec. 2.2's gating values replace the dense row for the column sums:
      // p / D on the token's top-k, 0 elsewhere (1/k each if D = 0).
      float *grow = (hier && !hier_here) ? a.gs + (size_t)t * N : nullptr;
      __syncwarp();
      for (int j = lane; j < N; j += 32) {
        prow_s[j] = 0.f;
        if (grow) grow[j] = 0.f;
      }
      __syncwarp();
      if (lane < k) {
        const float gv = (D > 0.f) ? __fdiv_rn(my_v, D) : __fdiv_rn(1.f, (float)k);
        prow_s[my_id] = gv;
        if (grow) grow[my_id] = gv;
      }
    }
  }
  __syncthreads();

  // ---- the chunk's column-sum tree (a4) ----
  // One chunk and no per-request step: the base set is final already, so
  // the selection's mask starts from it here and two barriers are saved.
  const bool one_pass = C == 1 && !hier;
  for (int j = tid; j < N; j += blockDim.x) {
    if (one_pass) s_mask[j] = s_base[j];
    float v[kChunk];
#pragma unroll
    for (int l = 0; l < kChunk; ++l) v[l] = ps[l * N + j];
#pragma unroll
    for (int o = kChunk / 2; o; o >>= 1) {
#pragma unroll
      for (int l = 0; l < o; ++l) v[l] = __fadd_rn(v[l], v[l + o]);
    }
    if (C == 1)
      s_col[j] = __fadd_rn(0.f, v[0]);  // one chunk: the batch sum is 0 + the chunk's tree
    else
      a.chunk_col[(size_t)c * N + j] = v[0];
  }

  // ---- HIER: Algorithm 3 for the requests inside this chunk ----
  if (hier_here) {
    const int T = a.T;
    for (int r = warp; r * T < nt; r += nwarps) {
      const int r0 = r * T, r1 = min(r0 + T, nt);
      float sc[kQ];
      uint32_t excl = 0;
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        const int j = lane + 32 * q;
        sc[q] = (j < N) ? canonical_sum(ps, N, j, r0, r1) : 0.f;
      }
      for (int x = r0; x < r1; ++x)
        for (int i = 0; i < a.k0; ++i) {
          const int e = s_top[x][i];
          if ((unsigned)e < (unsigned)N && (e & 31) == lane) {
            excl |= 1u << (e >> 5);
            s_base[e] = 1;
          }
        }
      LaneList<kQ> L;
      lane_load<kQ>(L, 0, N, lane, [&](int q, int) { return sc[q]; },
                    [&](int q, int) {
                      return ((excl >> q) & 1u) == 0 && (!a.sparse || sc[q] > 0.f);
                    });
      lane_sort<kQ>(L);
      lane_take<kQ>(L, a.m_r, [&](int, int id, float) {
        if (lane == 0) s_base[id] = 1;
      });
    }
  }
  __syncthreads();
  if (C > 1) {
    uint8_t *marks = a.chunk_marks + (size_t)c * 2 * N;
    for (int j = tid; j < N; j += blockDim.x) marks[j] = s_base[j];

    // ---- the last CTA to finish runs the selection ----
    __threadfence();
    __syncthreads();
    if (tid == 0) s_scal[0] = (atomicAdd(&a.done[0], 1) == C - 1) ? 1 : 0;
    __syncthreads();
    if (!s_scal[0]) return;
    __threadfence();

    for (int j = tid; j < N; j += blockDim.x) {
      float acc = 0.f;
      uint8_t b = 0;
      for (int cc = 0; cc < C; ++cc) {
        acc = __fadd_rn(acc, __ldcg(a.chunk_col + (size_t)cc * N + j));
        b |= __ldcg(a.chunk_marks + (size_t)cc * 2 * N + j);
      }
      s_col[j] = acc;
      s_base[j] = b;
    }
  }
  if (!one_pass) __syncthreads();

  if (hier && !hier_here) {
    // Requests cross chunk boundaries: Algorithm 3 from the full score matrix.
    const int T = a.T, R = B / T;
    for (int r = warp; r < R; r += nwarps) {
      const int r0 = r * T, r1 = r0 + T;
      float sc[kQ];
      uint32_t excl = 0;
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        const int j = lane + 32 * q;
        sc[q] = (j < N) ? canonical_sum(a.sparse ? a.gs : a.p, N, j, r0, r1) : 0.f;
      }
      for (int x = r0; x < r1; ++x)
        for (int i = 0; i < a.k0; ++i) {
          const int e = __ldcg(a.toptok + (size_t)x * kMaxK + i);
          if ((unsigned)e < (unsigned)N && (e & 31) == lane) {
            excl |= 1u << (e >> 5);
            s_base[e] = 1;
          }
        }
      LaneList<kQ> L;
      lane_load<kQ>(L, 0, N, lane, [&](int q, int) { return sc[q]; },
                    [&](int q, int) {
                      return ((excl >> q) & 1u) == 0 && (!a.sparse || sc[q] > 0.f);
                    });
      lane_sort<kQ>(L);
      lane_take<kQ>(L, a.m_r, [&](int, int id, float) {
        if (lane == 0) s_base[id] = 1;
      });
    }
    __syncthreads();
  }

  // ---- budgeted selection (a5) ----
  if (!one_pass) {
    for (int j = tid; j < N; j += blockDim.x) s_mask[j] = s_base[j];
    __syncthreads();
  }
  if (a.mode == XS_MODE_TOPK) {
    for (int j = tid; j < N; j += blockDim.x) s_mask[j] = 1;
  } else if (a.mode == XS_MODE_GROUP) {
    // Algorithm 5 runs whole rounds; after R rounds group g has added
    // min(R, avail_g) of its best remaining experts.  R* is the first round
    // count reaching m_g * G, or the one that exhausts every group.
    const int G = a.G, size = N / G;
    const int n_base = __syncthreads_count(tid < N && s_base[tid]);
    for (int g = warp; g < G; g += nwarps) {
      int cnt = 0;
      for (int j = g * size + lane; j < (g + 1) * size; j += 32)
        cnt += (s_base[j] == 0 && (!a.sparse || s_col[j] > 0.f)) ? 1 : 0;
      cnt = __reduce_add_sync(kFull, cnt);
      if (lane == 0) s_gl[g] = cnt;
    }
    __syncthreads();
    if (tid == 0) {
      int maxav = 0;
      for (int g = 0; g < G; ++g) maxav = max(maxav, s_gl[g]);
      const long long target = (long long)a.m_g * G;
      int R = 0;
      for (;;) {
        long long tot = n_base;
        for (int g = 0; g < G; ++g) tot += min(R, s_gl[g]);
        if (tot >= target || R >= maxav) break;
        ++R;
      }
      s_scal[1] = R;
    }
    __syncthreads();
    const int R = s_scal[1];
    if (R > 0)
      for (int g = warp; g < G; g += nwarps) {
        LaneList<kQ> L;
        lane_load<kQ>(L, g * size, size, lane, [&](int, int j) { return s_col[j]; },
                      [&](int, int j) { return s_base[j] == 0 && (!a.sparse || s_col[j] > 0.f); });
        lane_sort<kQ>(L);
        lane_take<kQ>(L, R, [&](int, int id, float) {
          if (lane == 0) s_mask[id] = 1;
        });
      }
  } else if (a.mode == XS_MODE_THRESH) {
    // Algorithm 1 in its threshold form: add the best remaining expert
    // while the covered mass f(S) is below tau f(E); by Proposition 1 adding
    // e adds scores[e] to f(S).
    if (warp == 0) {
      float vE[kQ], v0[kQ];
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        const int j = lane + 32 * q;
        vE[q] = (j < N) ? s_col[j] : 0.f;
        v0[q] = (j < N && s_base[j]) ? s_col[j] : 0.f;
      }
      const float target = __fmul_rn(a.tau, expert_tree<kQ>(vE));
      float f = expert_tree<kQ>(v0);
      LaneList<kQ> L;
      lane_load<kQ>(L, 0, N, lane, [&](int, int j) { return s_col[j]; },
                    [&](int, int j) { return s_base[j] == 0 && (!a.sparse || s_col[j] > 0.f); });
      lane_sort<kQ>(L);
      while (f < target) {
        float v = 0.f;
        int id = -1;
        if (lane_take<kQ>(L, 1, [&](int, int e, float sv) {
              id = e;
              v = sv;
            }) == 0)
          break;
        if (lane == 0) s_mask[id] = 1;
        f = __fadd_rn(f, v);
      }
    }
  } else if (warp == 0) {
    // BATCH (Algorithm 2) and the batch step of HIER (Algorithm 4): add the
    // `budget` best experts outside the base set by the batch column score.
    LaneList<kQ> L;
    lane_load<kQ>(L, 0, N, lane, [&](int, int j) { return s_col[j]; },
                  [&](int, int j) { return s_base[j] == 0 && (!a.sparse || s_col[j] > 0.f); });
    lane_mark_top<kQ>(L, a.budget, [&](int id) { s_mask[id] = 1; });
  }
  __syncthreads();

  // The router's status (if it reports one) rides on the barrier of the
  // selection statistics through a shared flag.  The token masks of the
  // small-batch permutation are cleared before that barrier too.
  if (C <= 2)
    for (int j = tid; j < N; j += blockDim.x) {
      s_cursor[j] = 0;
      s_counts[j] = 0;
    }
  int nsel, maxload;
  {
    int rs = 0;
    for (int i = tid; i < a.router_ctas; i += blockDim.x) rs |= __ldcg(a.router_status + i);
    if (rs != 0) s_rflag = 1;
  }
  if (a.G <= 1) {  // one group: its load is |S|
    nsel = __syncthreads_count(tid < N && s_mask[tid]);
    maxload = nsel;
  } else {
    if (tid == 0) s_gl[kMaxN] = 0;
    selection_stats(a, s_mask, s_gl, nsel, maxload);
  }
  const int rstat = s_rflag;
  // The mask, written by warp 0, then flagged (done[3]): the gather kernel,
  // resident already, warms L2 with the weights the gate/up kernel will
  // stream first while the refinement and permutation run.  The flag is a
  // hint, not a release: a reader that sees it before the mask only
  // prefetches other weights, so no fence slows this warp.
  if (warp == 0) {
    for (int j = lane; j < N; j += 32) a.mask[j] = s_mask[j];
    __syncwarp();
    if (lane == 0) *reinterpret_cast<volatile int32_t *>(a.done + 3) = 1;
  }
  if (tid == 0) {
    // Field by field: union_topk belongs to the union CTAs.
    Meta *m = a.meta;
    m->n_pairs = 0;
    m->n_tiles = 0;
    m->n_rows = 0;
    m->kprime = min(k, nsel);
    m->n_selected = nsel;
    m->n_used = 0;
    m->max_group_load = maxload;
    m->status = rstat ? XS_DEV_TIMEOUT : XS_DEV_OK;
  }
  if (!a.fuse_refine) return;
  // Small batches: refinement and permutation in this CTA too (no second
  // kernel); this chunk's scores are still in shared memory.  (The mask is
  // complete since the statistics' barrier; nothing the refinement writes
  // is read before it.)
  int32_t *ids_s = C == 1 ? &s_top[0][0] : nullptr;  // one chunk: ids stay in shared memory
  refine_tokens<kQ>(
      a, s_mask, nsel, s_chunk, s_tmp, 0, B, min(k, nsel),
      [&](int t) -> const float * {
        // The chunk's rows hold the sparse values in that mode; refine on dense p.
        return (t >= t0 && t < t0 + nt && !a.sparse) ? ps + (t - t0) * N : a.p + (size_t)t * N;
      },
      ids_s);
  if (C > 1) __threadfence();
  __syncthreads();
  static_assert(kFuseChunks <= 2, "the fused permutation takes at most two 32-token chunks");
  build_permutation_small(a, PermSmem{s_counts, s_cursor, s_chunk, s_tmp, s_scal, nullptr, nullptr},
                          ids_s);
}

template <int kQ>
__global__ void __launch_bounds__(kRouteThreads, 1) refine_kernel(RouteArgs a) {
  extern __shared__ int32_t s_wcnt[];   // [32][N] per-warp counts of the scatter (N <= 256)
  __shared__ uint8_t s_mask[kMaxN];
  __shared__ int32_t s_counts[kMaxN];
  __shared__ int32_t s_cursor[kMaxN];
  __shared__ int32_t s_chunk[kMaxN];
  __shared__ int32_t s_tmp[200];
  __shared__ int32_t s_scal[4];

  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x;
  const int B = a.B, N = a.N;
  const int C = chunk_count(B), c = blockIdx.x;
  const int t0 = c * kChunk, nt = min(kChunk, B - t0);
  const int kp = a.meta->kprime;
  for (int j = tid; j < N; j += blockDim.x) s_mask[j] = a.mask[j];
  __syncthreads();
  refine_tokens<kQ>(a, s_mask, a.meta->n_selected, s_chunk, s_tmp, t0, t0 + nt, kp,
                    [&](int t) { return a.p + (size_t)t * N; });

  // ---- the last CTA to finish builds the permutation (a7) ----
  __threadfence();
  __syncthreads();
  if (tid == 0) s_scal[0] = (atomicAdd(&a.done[1], 1) == C - 1) ? 1 : 0;
  __syncthreads();
  if (!s_scal[0]) return;
  __threadfence();
  build_permutation(a, PermSmem{s_counts, s_cursor, s_chunk, s_tmp, s_scal, s_wcnt, nullptr});
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
    int N, int d, int32_t *__restrict__ done) {
  __shared__ float red[kRtWarps][kRtOut];
  pdl_wait();
  pdl_trigger();
  if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x < 4) done[threadIdx.x] = 0;
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

// L2 warm-up for the gate/up kernel (packed weights).  Its stream-K split
// and segment order are those of ffn_tc.cu, predicted from the selected set
// (one tile per selected expert, in expert order): CTA c of G = ffn_ctas()
// takes steps [I c / G, I (c + 1) / G) of I = |S| x MT x KI and does first
// the steps of its last unit (if that unit continues in CTA c + 1), then
// those of its first unit (if it began in CTA c - 1), then its whole units.
// The first pf_bytes of that order are prefetched into L2, by the first
// kGatherWarmBlocks blocks (a few gate/up CTAs' ranges each: fewer blocks
// waiting on the flag and a less bursty stream of prefetches measured
// faster than one block per gate/up CTA).  A wrong prediction (an expert of
// S with no token, or more than one tile) only prefetches other weights.
__device__ void warm_gate_up(const GatherPf &g, int32_t *s_sel, int *s_n) {
  const int tid = threadIdx.x, lane = tid & 31;
  if (tid == 0) *s_n = -1;
  __syncthreads();
  if (tid < 32) {
    // Wait (bounded: 2 ms, a hint only) for the selection kernel's mask.
    bool ok = false;
    if (lane == 0) {
      const volatile int32_t *flag = g.ready;
      ok = *flag != 0;
      if (!ok) {
        const unsigned long long t0 = gtimer();
        while (!ok && gtimer() - t0 < 2000000ull) {
          __nanosleep(256);
          ok = *flag != 0;
        }
      }
    }
    ok = __shfl_sync(kFull, ok ? 1 : 0, 0) != 0;
    if (ok) {
      int n = 0;
      for (int j0 = 0; j0 < g.N; j0 += 32) {
        const bool sel = j0 + lane < g.N && __ldcg(g.mask + j0 + lane) != 0;
        const unsigned b = __ballot_sync(kFull, sel);
        if (sel) s_sel[n + __popc(b & ((1u << lane) - 1u))] = j0 + lane;
        n += __popc(b);
      }
      if (lane == 0) *s_n = n;
    }
  }
  __syncthreads();
  const int nS = *s_n;
  if (nS <= 0) return;
  const long long KI = g.KI, I = static_cast<long long>(nS) * g.MT * KI;
  const int G = ffn_ctas(static_cast<long long>(nS) * g.MT, g.KI, g.grid);  // gate/up CTAs
  const int n_steps = g.pf_bytes / g.stage_bytes;
  const int nb = gridDim.x < kGatherWarmBlocks ? static_cast<int>(gridDim.x) : kGatherWarmBlocks;
  for (int c = blockIdx.x; c < G; c += nb) {
    const long long ib = I * c / G, ie = I * (c + 1) / G;
    const long long uf = ib / KI, ul = (ie - 1) / KI;
    const long long kT0 = ib - uf * KI, kH1 = ie - ul * KI;
    // The i-th step of the CTA's order, for i < n_steps (thread i issues it).
    for (int i = tid; i < n_steps && i < ie - ib; i += blockDim.x) {
      long long st;
      if (uf == ul) {
        st = ib + i;
      } else {
        const long long nH = kH1 < KI ? kH1 : 0, nT = kT0 > 0 ? KI - kT0 : 0;
        if (i < nH)
          st = ul * KI + i;
        else if (i < nH + nT)
          st = ib + (i - nH);
        else
          st = (uf + (kT0 > 0 ? 1 : 0)) * KI + (i - nH - nT);
      }
      const long long u = st / KI;
      const int kk = static_cast<int>(st - u * KI);
      const int e = s_sel[u / g.MT], mt = static_cast<int>(u % g.MT);
      const uint8_t *blk =
          g.pk + ((static_cast<size_t>(e) * g.MT + mt) * g.KI + kk) * static_cast<size_t>(g.stage_bytes);
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(blk)),
                   "r"(g.stage_bytes)
                   : "memory");
    }
  }
}

// Xp[row] = x[token of pair perm[row]], 16-byte vectors, for the rows this
// call's FFN computes; with expert parallelism the other rows of zero_out
// (computed by other ranks) are set to zero instead.  Before that (packed
// weights), the gate/up kernel's first weights are brought into L2 as soon
// as the selected set is published.
__global__ void __launch_bounds__(256) gather_kernel(const uint16_t *__restrict__ x,
                                                     const int32_t *__restrict__ perm,
                                                     const Meta *__restrict__ meta,
                                                     uint16_t *__restrict__ xp,
                                                     float *__restrict__ zero_out, int B, int d,
                                                     int k, GatherPf pf) {
  __shared__ int32_t s_sel[kMaxN];
  __shared__ int s_n;
  if (pf.pk != nullptr && static_cast<int>(blockIdx.x) < kGatherWarmBlocks) warm_gate_up(pf, s_sel, &s_n);
  pdl_wait();
  pdl_trigger();
  const int row = blockIdx.x;
  const int P = meta->n_pairs;
  if (row >= meta->n_rows) return;
  const bool mine = row < P ? (row >= meta->row0 && row < meta->row1) : meta->srows != 0;
  if (!mine) {
    if (zero_out != nullptr) {
      float4 *dst = reinterpret_cast<float4 *>(zero_out + static_cast<size_t>(row) * d);
      for (int i = threadIdx.x; i < d / 4; i += blockDim.x) dst[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    return;
  }
  const int t = row < P ? perm[row] / k : (row - P) % B;  // routed pair, else shared row
  const uint4 *src = reinterpret_cast<const uint4 *>(x + (size_t)t * d);
  uint4 *dst = reinterpret_cast<uint4 *>(xp + (size_t)row * d);
  for (int i = threadIdx.x; i < d / 8; i += blockDim.x) dst[i] = __ldg(src + i);
}

// ---- a9: y_t = [x_t +] sum over slots s < k' of w_ts * out[pos(t, s)]
//              + sum over shared experts j of out[n_pairs + j * B + t], fp32, bf16 once.
// The residual x_t is added first when `resid` is given (layer stacks).
__global__ void __launch_bounds__(256) combine_kernel(const float *__restrict__ out,
                                                      const int32_t *__restrict__ pos,
                                                      const float *__restrict__ w,
                                                      const Meta *__restrict__ meta,
                                                      const uint16_t *__restrict__ resid,
                                                      uint16_t *__restrict__ y, int B, int d,
                                                      int k, int n_shared) {
  __shared__ int32_t s_row[kMaxK];
  __shared__ float s_w[kMaxK];
  __shared__ int32_t s_kp, s_pairs;
  const int t = blockIdx.y;
  const int c4 = blockIdx.x * blockDim.x + threadIdx.x;
  // Before pdl_wait(): the token's rows and weights and the pair count,
  // written by the routing kernels four launches earlier (complete before
  // this grid started), and x_t (an input, or the previous layer's output);
  // only `out` comes from the kernel just before.
  if (threadIdx.x < kMaxK) {
    const int s = threadIdx.x;
    s_row[s] = s < k ? __ldcg(pos + (size_t)t * k + s) : -1;
    s_w[s] = s < k ? __ldcg(w + (size_t)t * k + s) : 0.f;
  }
  if (threadIdx.x == 0) {
    s_kp = __ldcg(&meta->kprime);
    s_pairs = __ldcg(&meta->n_pairs);
  }
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  if (resid != nullptr && c4 < d / 4) {
    const uint2 r = __ldcg(reinterpret_cast<const uint2 *>(resid + (size_t)t * d) + c4);
    acc.x = __uint_as_float(r.x << 16);
    acc.y = __uint_as_float(r.x & 0xffff0000u);
    acc.z = __uint_as_float(r.y << 16);
    acc.w = __uint_as_float(r.y & 0xffff0000u);
  }
  __syncthreads();
  pdl_wait();
  pdl_trigger();
  if (c4 >= d / 4) return;
  const int kp = s_kp;
  for (int s = 0; s < kp; ++s) {
    const int r = s_row[s];
    if (r < 0) continue;  // only with non-finite scores
    const float ws = s_w[s];
    const float4 o = reinterpret_cast<const float4 *>(out + (size_t)r * d)[c4];
    acc.x = fmaf(ws, o.x, acc.x);
    acc.y = fmaf(ws, o.y, acc.y);
    acc.z = fmaf(ws, o.z, acc.z);
    acc.w = fmaf(ws, o.w, acc.w);
  }
  for (int j = 0; j < n_shared; ++j) {
    const size_t r = (size_t)s_pairs + (size_t)j * B + t;
    const float4 o = reinterpret_cast<const float4 *>(out + r * d)[c4];
    acc.x += o.x;
    acc.y += o.y;
    acc.z += o.z;
    acc.w += o.w;
  }
  __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x, acc.y);
  __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z, acc.w);
  uint2 v;
  v.x = *reinterpret_cast<uint32_t *>(&lo);
  v.y = *reinterpret_cast<uint32_t *>(&hi);
  reinterpret_cast<uint2 *>(y + (size_t)t * d)[c4] = v;
}

}  // namespace

template <int kQ>
cudaError_t launch_route_q(const RouteArgs &a, cudaStream_t s) {
  const int C = (a.B + kChunk - 1) / kChunk;
  RouteArgs b = a;
  b.fuse_refine = C <= kFuseChunks ? 1 : 0;
  const int wcnt = a.N <= kScatterMaxN ? 32 * a.N * 4 : 0;
  const int dyn1 = kChunk * a.N * 4 + (b.fuse_refine ? wcnt : 0);
  cudaError_t e = cudaFuncSetAttribute(score_kernel<kQ>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, dyn1);
  if (e != cudaSuccess) return e;
  e = launch_pdl(score_kernel<kQ>, dim3(2 * C), dim3(kRouteThreads), (size_t)dyn1, s, b);
  if (e != cudaSuccess) return e;
  if (b.fuse_refine) {
    if (a.events != nullptr) e = cudaEventRecord(reinterpret_cast<cudaEvent_t>(a.events[0]), s);
    return e;
  }
  if (a.events != nullptr) {
    e = cudaEventRecord(reinterpret_cast<cudaEvent_t>(a.events[0]), s);
    if (e != cudaSuccess) return e;
  }
  e = cudaFuncSetAttribute(refine_kernel<kQ>, cudaFuncAttributeMaxDynamicSharedMemorySize, wcnt);
  if (e != cudaSuccess) return e;
  return launch_pdl(refine_kernel<kQ>, dim3(C), dim3(kRouteThreads), (size_t)wcnt, s, b);
}

cudaError_t launch_route(const RouteArgs &a, cudaStream_t s) {
  if (a.N <= 64) return launch_route_q<2>(a, s);
  if (a.N <= 128) return launch_route_q<4>(a, s);
  if (a.N <= 256) return launch_route_q<8>(a, s);
  return launch_route_q<32>(a, s);
}

cudaError_t launch_router_logits(const uint16_t *x, const float *Wg, float *h, int B, int N,
                                 int d, int32_t *done, cudaStream_t s) {
  dim3 grid((N + kRtExp - 1) / kRtExp, (B + kRtTok - 1) / kRtTok);
  return launch_pdl(router_logits_kernel, grid, dim3(kRtWarps * 32), 0, s, x, Wg, h, B, N, d,
                    done);
}

cudaError_t launch_gather(const uint16_t *x, const int32_t *perm, const Meta *meta,
                          uint16_t *xp, float *zero_out, int max_rows, int B, int d, int k,
                          const GatherPf &pf, cudaStream_t s) {
  return launch_pdl(gather_kernel, dim3(max_rows), dim3(256), 0, s, x, perm, meta, xp, zero_out, B,
                    d, k, pf);
}

cudaError_t launch_combine(const float *out, const int32_t *pos, const float *w,
                           const Meta *meta, const uint16_t *resid, uint16_t *y, int B, int d,
                           int k, int n_shared, cudaStream_t s) {
  dim3 grid((d / 4 + 255) / 256, B);
  return launch_pdl(combine_kernel, grid, dim3(256), 0, s, out, pos, w, meta, resid, y, B, d, k,
                    n_shared);
}

}  // namespace xs
