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

// Total order of every top-k and argmax: larger score first, equal scores ->
// lower expert index.
__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
  return va > vb || (va == vb && ia < ib);
}

// Warp-wide argmax of (v, i) under `better`; every lane gets the winner.
__device__ __forceinline__ void warp_argmax(float &v, int &i) {
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    float v2 = __shfl_xor_sync(kFull, v, o);
    int i2 = __shfl_xor_sync(kFull, i, o);
    if (better(v2, i2, v, i)) {
      v = v2;
      i = i2;
    }
  }
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

// Ranks the values a warp holds (lane l holds columns l + 32 q, q < kMaxQ,
// valid where bit q of `live` is set) and returns, best first, up to
// `count` expert ids through `emit(r, id)`; -1 ends the list early.
template <int kMaxQ, class Emit>
__device__ __forceinline__ void warp_rank(const float (&vals)[kMaxQ], unsigned live, int count,
                                          int N, int lane, Emit emit) {
  for (int r = 0; r < count; ++r) {
    float bv = -INFINITY;
    int bi = INT_MAX;
#pragma unroll
    for (int q = 0; q < kMaxQ; ++q)
      if ((live >> q) & 1u)
        if (better(vals[q], lane + 32 * q, bv, bi)) {
          bv = vals[q];
          bi = lane + 32 * q;
        }
    warp_argmax(bv, bi);
    if (bi >= N) return;  // fewer candidates than `count`
    if ((bi & 31) == lane) live &= ~(1u << (bi >> 5));
    emit(r, bi, bv);
  }
}

// The whole selection in one CTA (steps a2-a7):
//   1. per token (one warp each): dense softmax of the logits (or the given
//      scores) held in registers, then its ranked top-max(k, k0) over E, which
//      marks the plain top-k union and the warm-up set S_0;
//   2. canonical column sums (one thread per expert) and, for HIER, the
//      per-request selections of Algorithm 3 (one warp per request);
//   3. the budgeted selection (rank counting in shared memory);
//   4. per token the top-k' inside S with renormalised weights, counting the
//      pairs per expert on the way;
//   5. prefix sums, FFN tiles, and the stable scatter of the pairs.
// The score matrix and the ids are staged in shared memory when they fit.
template <int kMaxQ>
__global__ void __launch_bounds__(kRouteThreads, 1) route_kernel(RouteArgs a) {
  extern __shared__ float dsm[];
  __shared__ uint8_t s_mask[kMaxN];   // S
  __shared__ uint8_t s_base[kMaxN];   // S_0 (or the union of the S_r for HIER)
  __shared__ uint8_t s_union[kMaxN];  // union of plain top-k
  __shared__ float s_col[kMaxN];      // batch column scores
  __shared__ int32_t s_counts[kMaxN];
  __shared__ int32_t s_off[kMaxN + 1];
  __shared__ int32_t s_toff[kMaxN + 1];
  __shared__ int32_t s_avail[kMaxN];
  __shared__ int32_t s_scal[8];      // 3:R* 4:|U| 5:tiles

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = blockDim.x >> 5;
  const int B = a.B, N = a.N, k = a.k;
  const int kk = max(k, a.k0);  // ranked list length per token
  float *ps = a.p_smem ? dsm : nullptr;
  int32_t *ids_s = a.ids_smem ? reinterpret_cast<int32_t *>(dsm + (a.p_smem ? B * N : 0)) : nullptr;
  const float *P = ps ? ps : a.p;

  for (int j = tid; j < N; j += blockDim.x) {
    s_mask[j] = 0;
    s_base[j] = 0;
    s_union[j] = 0;
    s_counts[j] = 0;
  }
  if (tid < 8) s_scal[tid] = 0;
  if (a.zero_words != nullptr)
    for (int i = tid; i < a.zero_count; i += blockDim.x) a.zero_words[i] = 0;
  __syncthreads();

  // ---- 1. scores (a2) and per-token ranking over E (a3) ----
  for (int t = warp; t < B; t += nwarps) {
    float vals[kMaxQ];
    unsigned live = 0;
    if (a.logits != nullptr) {
      const float *hrow = a.logits + (size_t)t * N;
      float mx = -INFINITY;
#pragma unroll
      for (int q = 0; q < kMaxQ; ++q) {
        const int j = lane + 32 * q;
        vals[q] = (j < N) ? hrow[j] : -INFINITY;
        mx = fmaxf(mx, vals[q]);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, o));
      float sum = 0.f;
#pragma unroll
      for (int q = 0; q < kMaxQ; ++q) {
        vals[q] = (lane + 32 * q < N) ? expf(vals[q] - mx) : 0.f;
        sum = __fadd_rn(sum, vals[q]);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) sum = __fadd_rn(sum, __shfl_xor_sync(kFull, sum, o));
#pragma unroll
      for (int q = 0; q < kMaxQ; ++q) {
        const int j = lane + 32 * q;
        if (j < N) {
          vals[q] = __fdiv_rn(vals[q], sum);
          a.p[(size_t)t * N + j] = vals[q];
          if (ps) ps[t * N + j] = vals[q];
          live |= 1u << q;
        }
      }
    } else {
#pragma unroll
      for (int q = 0; q < kMaxQ; ++q) {
        const int j = lane + 32 * q;
        vals[q] = (j < N) ? a.p[(size_t)t * N + j] : -INFINITY;
        if (j < N) {
          if (ps) ps[t * N + j] = vals[q];
          live |= 1u << q;
        }
      }
    }
    const bool hier = a.mode == XS_MODE_HIER;
    int32_t *top = a.toptok + (size_t)t * kMaxK;
    warp_rank<kMaxQ>(vals, live, kk, N, lane, [&](int r, int id, float) {
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
  if (a.mode == XS_MODE_HIER) {
    const int T = a.T, R = B / T;
    for (int r = warp; r < R; r += nwarps) {
      const int r0 = r * T, r1 = r0 + T;
      float sc[kMaxQ];
      unsigned live = 0;
#pragma unroll
      for (int q = 0; q < kMaxQ; ++q) {
        const int j = lane + 32 * q;
        sc[q] = 0.f;
        if (j < N) {
          sc[q] = canonical_sum(P, N, j, r0, r1);
          live |= 1u << q;
        }
      }
      // S0_r: union of Top k0 over the request's tokens.
      for (int x = r0; x < r1; ++x)
        for (int i = 0; i < a.k0; ++i) {
          const int e = a.toptok[(size_t)x * kMaxK + i];
          if ((unsigned)e < (unsigned)N && (e & 31) == lane) {
            live &= ~(1u << (e >> 5));
            s_base[e] = 1;
          }
        }
      // S_r = S0_r + Top m_r(scores_r, E \ S0_r).
      warp_rank<kMaxQ>(sc, live, a.m_r, N, lane, [&](int, int id, float) {
        if (lane == 0) s_base[id] = 1;
      });
    }
  }
  __syncthreads();

  // ---- 3. budgeted selection (a5) ----
  if (a.mode == XS_MODE_GROUP) {
    const int size = N / a.G;
    const int n_base = __syncthreads_count(tid < N && s_base[tid]);
    for (int j = tid; j < N; j += blockDim.x) s_avail[j] = 0;
    __syncthreads();
    for (int j = tid; j < N; j += blockDim.x)
      if (!s_base[j]) atomicAdd(&s_avail[j / size], 1);
    __syncthreads();
    if (tid == 0) {
      // Algorithm 5 runs whole rounds; after R rounds group g has added
      // min(R, avail_g).  R* is the first round count reaching m_g * G.
      int maxav = 0;
      for (int g = 0; g < a.G; ++g) maxav = max(maxav, s_avail[g]);
      const long long target = (long long)a.m_g * a.G;
      int R = 0;
      for (;;) {
        long long tot = n_base;
        for (int g = 0; g < a.G; ++g) tot += min(R, s_avail[g]);
        if (tot >= target || R >= maxav) break;
        ++R;
      }
      s_scal[3] = R;
    }
    __syncthreads();
    const int R = s_scal[3];
    for (int j = tid; j < N; j += blockDim.x) {
      if (s_base[j]) {
        s_mask[j] = 1;
        continue;
      }
      const int g0 = (j / size) * size;
      int rank = 0;
      for (int i = g0; i < g0 + size; ++i)
        if (!s_base[i] && better(s_col[i], i, s_col[j], j)) ++rank;
      if (rank < R) s_mask[j] = 1;
    }
  } else if (a.mode == XS_MODE_TOPK) {
    for (int j = tid; j < N; j += blockDim.x) s_mask[j] = 1;
  } else {
    // BATCH (Algorithm 2) and the batch step of HIER (Algorithm 4): add the
    // `budget` best experts outside the base set by the batch column score.
    const int m = a.budget;
    for (int j = tid; j < N; j += blockDim.x) {
      if (s_base[j]) {
        s_mask[j] = 1;
        continue;
      }
      int rank = 0;
      for (int i = 0; i < N && rank < m; ++i)
        if (!s_base[i] && better(s_col[i], i, s_col[j], j)) ++rank;
      if (rank < m) s_mask[j] = 1;
    }
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
#pragma unroll
    for (int o = 16; o; o >>= 1) best = max(best, __shfl_xor_sync(kFull, best, o));
    if (lane == 0) s_scal[2] = best;
  }
  for (int j = tid; j < N; j += blockDim.x) a.mask[j] = s_mask[j];
  const int kp = min(k, nsel);

  // ---- 4. refinement (a6): Top k'(G_i, S), renormalised weights, pair counts ----
  for (int t = warp; t < B; t += nwarps) {
    float vals[kMaxQ];
    unsigned live = 0;
#pragma unroll
    for (int q = 0; q < kMaxQ; ++q) {
      const int j = lane + 32 * q;
      vals[q] = 0.f;
      if (j < N && s_mask[j]) {
        vals[q] = P[(size_t)t * N + j];
        live |= 1u << q;
      }
    }
    int my_id = -1;  // lane s keeps slot s
    float my_v = 0.f;
    float D = 0.f;
    int got = 0;
    warp_rank<kMaxQ>(vals, live, kp, N, lane, [&](int r, int id, float v) {
      if (lane == r) {
        my_id = id;
        my_v = v;
      }
      D = __fadd_rn(D, v);  // slot order, identical on every lane
      got = r + 1;
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
  const int P2 = B * k;
  if (warp == 0) {
    // Exclusive scans over N (<= 1024) of counts and of tile counts, per/lane each.
    const int per = (N + 31) / 32;
    int c_sum = 0, t_sum = 0, used = 0;
    for (int i = 0; i < per; ++i) {
      const int e = lane * per + i;
      if (e < N) {
        c_sum += s_counts[e];
        t_sum += (s_counts[e] + kTileTok - 1) / kTileTok;
        used += s_counts[e] > 0;
      }
    }
    int c_inc = c_sum, t_inc = t_sum, u_inc = used;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int c2 = __shfl_up_sync(kFull, c_inc, o), t2 = __shfl_up_sync(kFull, t_inc, o);
      const int u2 = __shfl_up_sync(kFull, u_inc, o);
      if (lane >= o) {
        c_inc += c2;
        t_inc += t2;
        u_inc += u2;
      }
    }
    int c_run = c_inc - c_sum, t_run = t_inc - t_sum;
    for (int i = 0; i < per; ++i) {
      const int e = lane * per + i;
      if (e < N) {
        s_off[e] = c_run;
        s_toff[e] = t_run;
        c_run += s_counts[e];
        t_run += (s_counts[e] + kTileTok - 1) / kTileTok;
      }
    }
    if (lane == 31) {
      s_off[N] = c_inc;
      s_toff[N] = t_inc;
      s_scal[4] = u_inc;
      s_scal[5] = t_inc;
    }
  }
  __syncthreads();
  for (int e = tid; e < N; e += blockDim.x) {
    const int c = s_counts[e];
    a.counts[e] = c;
    a.offsets[e] = s_off[e];
    if (a.counts_out) a.counts_out[e] = c;
    if (a.offsets_out) a.offsets_out[e] = s_off[e];
    for (int tt = 0; tt * kTileTok < c; ++tt) {
      Tile tl;
      tl.expert = e;
      tl.row0 = s_off[e] + tt * kTileTok;
      tl.ntok = min(kTileTok, c - tt * kTileTok);
      tl.pad = 0;
      a.tiles[s_toff[e] + tt] = tl;
    }
  }
  if (tid == 0) {
    a.offsets[N] = s_off[N];
    if (a.offsets_out) a.offsets_out[N] = s_off[N];
  }
  __syncthreads();
  if (warp == 0) {
    // s_counts becomes the running cursor of each expert (warp 0 only from here).
    for (int e = lane; e < N; e += 32) s_counts[e] = s_off[e];
    __syncwarp();
    const unsigned lt = (1u << lane) - 1u;
    const int32_t *ids = ids_s ? ids_s : a.ids;
    for (int base = 0; base < P2; base += 32) {
      const int q = base + lane;
      int e = (q < P2) ? ids[q] : -1;
      if ((unsigned)e >= (unsigned)N) e = -1;
      const unsigned peers = __match_any_sync(kFull, e);
      const int rank = __popc(peers & lt);
      const int old = (e >= 0) ? s_counts[e] : 0;
      __syncwarp();
      if (e >= 0) {
        const int r = old + rank;
        a.perm[r] = q;
        a.pos[q] = r;
        if (a.perm_out) a.perm_out[r] = q;
        if (rank == 0) s_counts[e] = old + __popc(peers);
      } else if (q < P2) {
        a.pos[q] = -1;
      }
      __syncwarp();
    }
    if (lane == 0) {
      Meta m;
      m.n_pairs = s_off[N];  // == B * kp unless scores were non-finite
      m.n_tiles = s_scal[5];
      m.kprime = kp;
      m.n_selected = nsel;
      m.n_used = s_scal[4];
      m.union_topk = n_union;
      m.max_group_load = s_scal[2];
      m.status = 0;
      for (int i = 0; i < 8; ++i) m.pad[i] = 0;
      *a.meta = m;
      if (a.stats) {
        xs_stats st;
        st.n_selected = nsel;
        st.n_used = s_scal[4];
        st.union_topk = n_union;
        st.max_group_load = s_scal[2];
        st.n_pairs = s_off[N];
        st.status = 0;
        st.reserved[0] = st.reserved[1] = 0;
        *a.stats = st;
      }
    }
  }
}

// ---- a1: router logits h = W_g x, fp32.
// A block owns 8 tokens x 8 experts; its 8 warps split the d dimension into 8
// contiguous slices.  A lane walks its slice in float4 steps and keeps the
// 8 x 8 outer-product sums in registers (each W_g and x value loaded once per
// block, 16 loads per 256 FMAs).  A butterfly reduce-scatter over the 32
// lanes leaves each lane two finished sums, and the 8 warp partials are
// added in warp order through shared memory: a fixed order, so h is
// reproducible bit for bit.
constexpr int kRtTok = 8;
constexpr int kRtExp = 8;
constexpr int kRtWarps = 8;
constexpr int kRtOut = kRtTok * kRtExp;   // 64 sums per lane before the reduction

__global__ void __launch_bounds__(kRtWarps * 32) router_logits_kernel(
    const uint16_t *__restrict__ x, const float *__restrict__ Wg, float *__restrict__ h, int B,
    int N, int d) {
  __shared__ float red[kRtWarps][kRtOut];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int e0 = blockIdx.x * kRtExp, t0 = blockIdx.y * kRtTok;
  const int d4 = d / 4;
  const int c_begin = warp * (d4 / kRtWarps), c_end = (warp + 1) * (d4 / kRtWarps);
  float acc[kRtOut];
#pragma unroll
  for (int i = 0; i < kRtOut; ++i) acc[i] = 0.f;
  const float4 *wbase = reinterpret_cast<const float4 *>(Wg);
  const uint2 *xbase = reinterpret_cast<const uint2 *>(x);
#pragma unroll 1
  for (int c4 = c_begin + lane; c4 < c_end; c4 += 32) {
    float xf[kRtTok][4];
#pragma unroll
    for (int j = 0; j < kRtTok; ++j) {
      uint2 v = make_uint2(0u, 0u);
      if (t0 + j < B) v = __ldg(xbase + (size_t)(t0 + j) * d4 + c4);
      xf[j][0] = __uint_as_float(v.x << 16);
      xf[j][1] = __uint_as_float(v.x & 0xffff0000u);
      xf[j][2] = __uint_as_float(v.y << 16);
      xf[j][3] = __uint_as_float(v.y & 0xffff0000u);
    }
#pragma unroll
    for (int e = 0; e < kRtExp; ++e) {
      float4 wv = make_float4(0.f, 0.f, 0.f, 0.f);
      if (e0 + e < N) wv = __ldg(wbase + (size_t)(e0 + e) * d4 + c4);
#pragma unroll
      for (int j = 0; j < kRtTok; ++j) {
        float a = acc[j * kRtExp + e];
        a = fmaf(xf[j][0], wv.x, a);
        a = fmaf(xf[j][1], wv.y, a);
        a = fmaf(xf[j][2], wv.z, a);
        a = fmaf(xf[j][3], wv.w, a);
        acc[j * kRtExp + e] = a;
      }
    }
  }
  // Reduce-scatter: after the step with offset o a lane keeps the half of its
  // values selected by bit o of its lane id; after five steps lane l holds
  // the complete sums of outputs 2l and 2l + 1.
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
  red[warp][2 * lane] = acc[0];
  red[warp][2 * lane + 1] = acc[1];
  __syncthreads();
  if (threadIdx.x < kRtOut) {
    float s = red[0][threadIdx.x];
#pragma unroll
    for (int w = 1; w < kRtWarps; ++w) s += red[w][threadIdx.x];
    const int t = t0 + threadIdx.x / kRtExp, e = e0 + threadIdx.x % kRtExp;
    if (t < B && e < N) h[(size_t)t * N + e] = s;
  }
}

// Xp[row] = x[token of pair perm[row]], 16-byte vectors.
__global__ void __launch_bounds__(256) gather_kernel(const uint16_t *__restrict__ x,
                                                     const int32_t *__restrict__ perm,
                                                     const Meta *__restrict__ meta,
                                                     uint16_t *__restrict__ xp, int d, int k) {
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
  return (*p_smem ? p_bytes : 0) + (*ids_smem ? ids_bytes : 0);
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
  route_kernel<kMaxQ><<<1, kRouteThreads, dyn, s>>>(a);
  return cudaGetLastError();
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
  router_logits_kernel<<<grid, kRtWarps * 32, 0, s>>>(x, Wg, h, B, N, d);
  return cudaGetLastError();
}

cudaError_t launch_gather(const uint16_t *x, const int32_t *perm, const Meta *meta,
                          uint16_t *xp, int max_pairs, int d, int k, cudaStream_t s) {
  gather_kernel<<<max_pairs, 256, 0, s>>>(x, perm, meta, xp, d, k);
  return cudaGetLastError();
}

cudaError_t launch_combine(const float *out, const int32_t *pos, const float *w,
                           const Meta *meta, uint16_t *y, int B, int d, int k,
                           cudaStream_t s) {
  dim3 grid((d / 4 + 255) / 256, B);
  combine_kernel<<<grid, 256, 0, s>>>(out, pos, w, meta, y, d, k);
  return cudaGetLastError();
}

}  // namespace xs
