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

// One warp ranks the experts of row `t` of p: writes the `count` best of E,
// best first, to out[0..count).  kMaxQ = columns held per lane (N <= 32 kMaxQ).
template <int kMaxQ>
__device__ void warp_row_top(const float *__restrict__ prow, int N, int count,
                             int32_t *__restrict__ out, int lane) {
  float vals[kMaxQ];
  unsigned live = 0;
#pragma unroll
  for (int q = 0; q < kMaxQ; ++q) {
    int j = lane + 32 * q;
    vals[q] = (j < N) ? prow[j] : -INFINITY;
    if (j < N) live |= 1u << q;
  }
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
    if (bi >= N) bi = -1;  // only with non-finite scores
    if (bi >= 0 && (bi & 31) == lane) live &= ~(1u << (bi >> 5));
    if (lane == 0) out[r] = bi;
  }
}

template <int kMaxQ>
__global__ void __launch_bounds__(kRouteThreads, 1) route_kernel(RouteArgs a) {
  __shared__ uint8_t s_mask[kMaxN];   // S
  __shared__ uint8_t s_base[kMaxN];   // S_0 (or the union of the S_r for HIER)
  __shared__ uint8_t s_union[kMaxN];  // union of plain top-k
  __shared__ float s_col[kMaxN];      // batch column scores
  __shared__ int32_t s_counts[kMaxN];
  __shared__ int32_t s_off[kMaxN + 1];
  __shared__ int32_t s_toff[kMaxN + 1];
  __shared__ int32_t s_cursor[kMaxN];
  __shared__ int32_t s_avail[kMaxN];
  __shared__ int32_t s_scal[8];      // 0:|S| 1:union 2:maxload 3:R* 4:|U| 5:tiles 6:|S_0|

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = blockDim.x >> 5;
  const int B = a.B, N = a.N, k = a.k;
  const int kk = max(k, a.k0);  // ranked list length per token

  // ---- a2: dense softmax over all N experts (if logits are given) ----
  if (a.logits != nullptr) {
    for (int t = warp; t < B; t += nwarps) {
      const float *h = a.logits + (size_t)t * N;
      float mx = -INFINITY;
      for (int j = lane; j < N; j += 32) mx = fmaxf(mx, h[j]);
#pragma unroll
      for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, o));
      float sum = 0.f;
      for (int j = lane; j < N; j += 32) sum = __fadd_rn(sum, expf(h[j] - mx));
#pragma unroll
      for (int o = 16; o; o >>= 1) sum = __fadd_rn(sum, __shfl_xor_sync(kFull, sum, o));
      for (int j = lane; j < N; j += 32) a.p[(size_t)t * N + j] = __fdiv_rn(expf(h[j] - mx), sum);
    }
  }
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

  // ---- a3: per-token ranked top-kk over E (warm-up and plain top-k union) ----
  for (int t = warp; t < B; t += nwarps)
    warp_row_top<kMaxQ>(a.p + (size_t)t * N, N, kk, a.toptok + (size_t)t * kMaxK, lane);
  __syncthreads();
  for (int t = tid; t < B; t += blockDim.x) {
    const int32_t *row = a.toptok + (size_t)t * kMaxK;
    for (int r = 0; r < k; ++r)
      if ((unsigned)row[r] < (unsigned)N) s_union[row[r]] = 1;
    if (a.mode != XS_MODE_HIER)
      for (int r = 0; r < a.k0; ++r)
        if ((unsigned)row[r] < (unsigned)N) s_base[row[r]] = 1;
  }
  // ---- a4: batch column scores ----
  for (int j = tid; j < N; j += blockDim.x) s_col[j] = canonical_sum(a.p, N, j, 0, B);
  __syncthreads();

  // ---- a5': HIER per-request selection (Algorithm 3), one warp per request ----
  if (a.mode == XS_MODE_HIER) {
    const int T = a.T, R = B / T;
    for (int r = warp; r < R; r += nwarps) {
      const int r0 = r * T, r1 = r0 + T;
      float sc[kMaxQ];
      unsigned live = 0;
#pragma unroll
      for (int q = 0; q < kMaxQ; ++q) {
        int j = lane + 32 * q;
        sc[q] = 0.f;
        if (j < N) {
          sc[q] = canonical_sum(a.p, N, j, r0, r1);
          live |= 1u << q;
        }
      }
      // S0_r: union of Top k0 over the request's tokens.
      for (int x = r0; x < r1; ++x)
        for (int i = 0; i < a.k0; ++i) {
          int e = a.toptok[(size_t)x * kMaxK + i];
          if ((unsigned)e < (unsigned)N && (e & 31) == lane) {
            live &= ~(1u << (e >> 5));
            s_base[e] = 1;
          }
        }
      // S_r = S0_r + Top m_r(scores_r, E \ S0_r).
      for (int c = 0; c < a.m_r; ++c) {
        float bv = -INFINITY;
        int bi = INT_MAX;
#pragma unroll
        for (int q = 0; q < kMaxQ; ++q)
          if ((live >> q) & 1u)
            if (better(sc[q], lane + 32 * q, bv, bi)) {
              bv = sc[q];
              bi = lane + 32 * q;
            }
        warp_argmax(bv, bi);
        if (bi >= N) break;
        if ((bi & 31) == lane) {
          live &= ~(1u << (bi >> 5));
          s_base[bi] = 1;
        }
      }
    }
    __syncthreads();
  }

  // ---- a5: budgeted selection ----
  for (int j = tid; j < N; j += blockDim.x)
    if (s_base[j]) atomicAdd(&s_scal[6], 1);
  if (a.mode == XS_MODE_GROUP) {
    for (int j = tid; j < N; j += blockDim.x) s_avail[j] = 0;
    __syncthreads();
    const int size = N / a.G;
    for (int j = tid; j < N; j += blockDim.x)
      if (!s_base[j]) atomicAdd(&s_avail[j / size], 1);
    __syncthreads();
    if (tid == 0) {
      // Algorithm 5 runs whole rounds; after R rounds group g has added
      // min(R, avail_g).  R* is the first round count reaching m_g * G.
      int maxav = 0;
      for (int g = 0; g < a.G; ++g) maxav = max(maxav, s_avail[g]);
      long long target = (long long)a.m_g * a.G;
      int R = 0;
      for (;;) {
        long long tot = s_scal[6];
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
  {
    const int G = a.G >= 1 ? a.G : 1;
    const int size = N / G;
    for (int j = tid; j < N; j += blockDim.x) {
      if (s_mask[j]) atomicAdd(&s_scal[0], 1);
      if (s_union[j]) atomicAdd(&s_scal[1], 1);
    }
    if (warp == 0) {
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
  }
  for (int j = tid; j < N; j += blockDim.x) a.mask[j] = s_mask[j];
  __syncthreads();
  const int nsel = s_scal[0];
  const int kp = min(k, nsel);

  // ---- a6: refinement, Top k'(G_i, S) with renormalised weights ----
  for (int t = warp; t < B; t += nwarps) {
    const float *prow = a.p + (size_t)t * N;
    float vals[kMaxQ];
    unsigned live = 0;
#pragma unroll
    for (int q = 0; q < kMaxQ; ++q) {
      int j = lane + 32 * q;
      vals[q] = 0.f;
      if (j < N && s_mask[j]) {
        vals[q] = prow[j];
        live |= 1u << q;
      }
    }
    int my_id = -1;      // lane s keeps slot s
    float my_v = 0.f;
    float D = 0.f;
    for (int s = 0; s < kp; ++s) {
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
      if (bi >= N) bi = -1;  // only with non-finite scores
      if (bi >= 0 && (bi & 31) == lane) live &= ~(1u << (bi >> 5));
      if (lane == s) {
        my_id = bi;
        my_v = bv;
      }
      D = __fadd_rn(D, bv);  // slot order, identical on every lane
    }
    if (lane < k) {
      float wv = 0.f;
      if (lane < kp) wv = (D > 0.f) ? __fdiv_rn(my_v, D) : __fdiv_rn(1.f, (float)kp);
      a.ids[(size_t)t * k + lane] = (lane < kp) ? my_id : -1;
      a.w[(size_t)t * k + lane] = wv;
    }
  }
  __syncthreads();

  // ---- a7: permutation (counting sort by expert, stable in (token, slot)) ----
  const int P = B * k;
  for (int q = tid; q < P; q += blockDim.x) {
    int e = a.ids[q];
    if ((unsigned)e < (unsigned)N) atomicAdd(&s_counts[e], 1);
  }
  __syncthreads();
  if (warp == 0) {
    // Exclusive scans over N (<= 1024) of counts and of tile counts, 32 per lane.
    const int per = (N + 31) / 32;
    int c_sum = 0, t_sum = 0, used = 0;
    for (int i = 0; i < per; ++i) {
      int e = lane * per + i;
      if (e < N) {
        c_sum += s_counts[e];
        t_sum += (s_counts[e] + kTileTok - 1) / kTileTok;
        used += s_counts[e] > 0;
      }
    }
    int c_inc = c_sum, t_inc = t_sum, u_inc = used;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int c2 = __shfl_up_sync(kFull, c_inc, o), t2 = __shfl_up_sync(kFull, t_inc, o);
      int u2 = __shfl_up_sync(kFull, u_inc, o);
      if (lane >= o) {
        c_inc += c2;
        t_inc += t2;
        u_inc += u2;
      }
    }
    int c_run = c_inc - c_sum, t_run = t_inc - t_sum;
    for (int i = 0; i < per; ++i) {
      int e = lane * per + i;
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
    s_cursor[e] = s_off[e];
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
    const unsigned lt = (1u << lane) - 1u;
    for (int base = 0; base < P; base += 32) {
      const int q = base + lane;
      int e = (q < P) ? a.ids[q] : -1;
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
      } else if (q < P) {
        a.pos[q] = -1;
      }
      __syncwarp();
    }
  }
  if (tid == 0) {
    Meta m;
    m.n_pairs = s_off[N];  // == B * kp unless scores were non-finite
    m.n_tiles = s_scal[5];
    m.kprime = kp;
    m.n_selected = nsel;
    m.n_used = s_scal[4];
    m.union_topk = s_scal[1];
    m.max_group_load = s_scal[2];
    m.status = 0;
    for (int i = 0; i < 8; ++i) m.pad[i] = 0;
    *a.meta = m;
    if (a.stats) {
      xs_stats st;
      st.n_selected = nsel;
      st.n_used = s_scal[4];
      st.union_topk = s_scal[1];
      st.max_group_load = s_scal[2];
      st.n_pairs = s_off[N];
      st.status = 0;
      st.reserved[0] = st.reserved[1] = 0;
      *a.stats = st;
    }
  }
}

// ---- a1: router logits h = W_g x, fp32.  Block = 8 experts x 8 tokens; warp
// w owns expert e0 + w; a lane sums its slice of d (float4 steps), then the
// warp adds the 32 lane sums with a butterfly.
constexpr int kRtTok = 8;
constexpr int kRtExp = 8;

__global__ void __launch_bounds__(256) router_logits_kernel(const uint16_t *__restrict__ x,
                                                            const float *__restrict__ Wg,
                                                            float *__restrict__ h, int B,
                                                            int N, int d) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int e = blockIdx.x * kRtExp + warp;
  const int t0 = blockIdx.y * kRtTok;
  float acc[kRtTok];
#pragma unroll
  for (int j = 0; j < kRtTok; ++j) acc[j] = 0.f;
  if (e < N) {
    const float4 *wrow = reinterpret_cast<const float4 *>(Wg + (size_t)e * d);
    for (int c4 = lane; c4 < d / 4; c4 += 32) {
      const float4 wv = __ldg(wrow + c4);
#pragma unroll
      for (int j = 0; j < kRtTok; ++j) {
        if (t0 + j < B) {
          const uint2 xv = __ldg(reinterpret_cast<const uint2 *>(x + (size_t)(t0 + j) * d) + c4);
          const float x0 = __uint_as_float(xv.x << 16), x1 = __uint_as_float(xv.x & 0xffff0000u);
          const float x2 = __uint_as_float(xv.y << 16), x3 = __uint_as_float(xv.y & 0xffff0000u);
          acc[j] = fmaf(x0, wv.x, acc[j]);
          acc[j] = fmaf(x1, wv.y, acc[j]);
          acc[j] = fmaf(x2, wv.z, acc[j]);
          acc[j] = fmaf(x3, wv.w, acc[j]);
        }
      }
    }
  }
#pragma unroll
  for (int j = 0; j < kRtTok; ++j)
#pragma unroll
    for (int o = 16; o; o >>= 1) acc[j] += __shfl_xor_sync(kFull, acc[j], o);
  if (e < N) {
    float mine = 0.f;
#pragma unroll
    for (int j = 0; j < kRtTok; ++j)
      if (lane == j) mine = acc[j];
    if (lane < kRtTok && t0 + lane < B) h[(size_t)(t0 + lane) * N + e] = mine;
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

cudaError_t launch_route(const RouteArgs &a, cudaStream_t s) {
  if (a.N <= 64)
    route_kernel<2><<<1, kRouteThreads, 0, s>>>(a);
  else if (a.N <= 128)
    route_kernel<4><<<1, kRouteThreads, 0, s>>>(a);
  else if (a.N <= 256)
    route_kernel<8><<<1, kRouteThreads, 0, s>>>(a);
  else
    route_kernel<32><<<1, kRouteThreads, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_router_logits(const uint16_t *x, const float *Wg, float *h, int B, int N,
                                 int d, cudaStream_t s) {
  dim3 grid((N + kRtExp - 1) / kRtExp, (B + kRtTok - 1) / kRtTok);
  router_logits_kernel<<<grid, 256, 0, s>>>(x, Wg, h, B, N, d);
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
