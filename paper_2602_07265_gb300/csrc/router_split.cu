// Router logits h = W_g x (step a1, Sec. 2.2) on the CUDA cores for decode
// batches (B < 64), in fp32: the layer's x is bf16 and the router weights
// are fp32, and each logit is a d-long dot product.
//
// At these batch sizes the work is 2 B N d flops, far below what the SMs do
// in a microsecond, so the kernel is bound by moving W_g (N d 4 bytes, read
// once) and x through the SMs.  A CTA owns 8 experts, up to 32 tokens and one
// of S slices of d (64-column chunks), so every SM has work, each W_g row
// slice is read by one CTA per 32 tokens, and x by one CTA per 8 experts.
// Its W_g rows are requested with bulk copies before griddepcontrol.wait
// (the weights do not depend on the kernel before) and its x rows right
// after it, all into shared memory at once; the CTA then reads only shared
// memory.
//
// Arithmetic: a lane owns 8 experts x 4 tokens and one of four column sets;
// the eight warps take interleaved 16-column blocks.  Products are
// accumulated with packed fp32 FMAs (__ffma2_rn) in two interleaved partial
// sums per output (even and odd columns), which the lane then adds; the four
// column sets are added with a butterfly over lanes and the eight warps in
// warp order through shared memory.  Every order is fixed, so the slice sums
// are reproducible bit for bit.  Slice s is written to h[s][t][e]; the
// selection kernel adds the S slices in order s = 0 .. S-1 when it loads a
// token's logits.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "tc_ptx.cuh"
#include "xs_internal.cuh"

namespace xs {
namespace {

using namespace ptx;

constexpr int kRsThreads = 256;
constexpr int kRsWarps = kRsThreads / 32;
constexpr int kRsEB = 8;                   // experts per CTA
constexpr int kRsChunk = 64;               // columns per slicing unit
constexpr int kRsMaxDS = 32 * kRsChunk;    // columns per slice at most (shared memory)
constexpr int kRsMaxSplits = 4;            // slices the selection kernel adds, unless d needs more
                                           // (up to 8: d <= kRouterSplitMaxD)
constexpr int kRsSub = 1;                  // sub-chunks of a slice, each with its own barrier
constexpr int kRsPad = 32;                 // x row padding in shared memory (bank spread)
constexpr uint64_t kRsWaitNs = 1000000000ull;

// Tokens per CTA for kTI token groups of 8 per lane.
__host__ __device__ constexpr int rs_tb(int kTI) { return 8 * kTI; }

// Barriers, W tile [8][DS] fp32, x tile [TB][DS] bf16 (padded rows); the
// cross-warp sums reuse the space from the W tile on ([8 warps][TB][8]).
__host__ __device__ constexpr size_t rs_smem_bytes(int DS, int TB) {
  const size_t tiles = static_cast<size_t>(kRsEB) * DS * 4 + static_cast<size_t>(TB) * (2 * DS + kRsPad);
  const size_t red = static_cast<size_t>(kRsWarps) * TB * kRsEB * 4;
  return 64 + (tiles > red ? tiles : red);
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

template <int kTI>
__global__ void __launch_bounds__(kRsThreads, 1)
    router_split_kernel(const uint16_t *__restrict__ x, const float *__restrict__ Wg,
                        float *__restrict__ h, int B, int N, int d, int S,
                        int32_t *__restrict__ done, int32_t *__restrict__ status) {
  constexpr int TB = rs_tb(kTI);
  constexpr int V = kRsEB * kTI;  // sums per lane before the column sets are added
  extern __shared__ __align__(16) uint8_t rs_smem[];
  __shared__ int s_ok;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int e0 = blockIdx.x * kRsEB, s = blockIdx.y, t0 = blockIdx.z * TB;
  const int nch = d / kRsChunk;
  const int u0 = nch * s / S, nu = nch * (s + 1) / S - u0;  // this slice's 64-column units
  const int c0 = u0 * kRsChunk, DS = nu * kRsChunk;
  const int ne = min(kRsEB, N - e0), nt = min(TB, B - t0);
  const int xstride = 2 * DS + kRsPad;  // bytes per x row in shared memory
  const uint32_t bar0 = smem_u32(rs_smem);
  float *Ws = reinterpret_cast<float *>(rs_smem + 64);
  uint8_t *xs = rs_smem + 64 + static_cast<size_t>(kRsEB) * DS * 4;
  const int cta = (blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
  // Sub-chunk q covers units [sub(q), sub(q + 1)) of the slice.
  auto sub = [&](int q) { return nu * q / kRsSub; };

  if (threadIdx.x == 0) {
    for (int q = 0; q < kRsSub; ++q) {
      const int w = (sub(q + 1) - sub(q)) * kRsChunk;  // columns
      mbar_init(bar0 + 8 * q, 1);
      fence_mbar_init();
      mbar_arrive_expect_tx(bar0 + 8 * q, static_cast<uint32_t>((ne * 4 + nt * 2) * w));
    }
  }
  __syncthreads();
  // W_g does not depend on the kernel before: its rows are requested first,
  // one bulk copy per (expert, sub-chunk), spread over the lanes of warp 0.
  if (warp == 0) {
    const uint64_t pol_w = policy_evict_first();
    for (int i = lane; i < ne * kRsSub; i += 32) {
      const int e = i / kRsSub, q = i % kRsSub;
      const int ca = sub(q) * kRsChunk, w = (sub(q + 1) - sub(q)) * kRsChunk;
      if (w > 0)
        bulk_load(smem_u32(Ws + static_cast<size_t>(e) * DS + ca),
                  Wg + static_cast<size_t>(e0 + e) * d + c0 + ca, w * 4, bar0 + 8 * q, pol_w);
    }
  }
  pdl_wait();
  pdl_trigger();
  if (cta == 0 && threadIdx.x < 4) done[threadIdx.x] = 0;
  if (warp == 0) {
    const uint64_t pol_x = policy_evict_last();  // every expert block reads these rows
    for (int i = lane; i < nt * kRsSub; i += 32) {
      const int t = i / kRsSub, q = i % kRsSub;
      const int ca = sub(q) * kRsChunk, w = (sub(q + 1) - sub(q)) * kRsChunk;
      if (w > 0)
        bulk_load(smem_u32(xs + static_cast<size_t>(t) * xstride + ca * 2),
                  x + static_cast<size_t>(t0 + t) * d + c0 + ca, w * 2, bar0 + 8 * q, pol_x);
    }
  }
  // Rows past N or B read as zeros (no copy writes them).
  for (int r = ne; r < kRsEB; ++r)
    for (int i = threadIdx.x; i < DS / 4; i += kRsThreads)
      reinterpret_cast<float4 *>(Ws + static_cast<size_t>(r) * DS)[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int r = nt; r < TB; ++r)
    for (int i = threadIdx.x; i < DS / 8; i += kRsThreads)
      reinterpret_cast<uint4 *>(xs + static_cast<size_t>(r) * xstride)[i] = make_uint4(0u, 0u, 0u, 0u);
  __syncthreads();

  // Lane (cs, tg): column set cs = lane / 8 (4 columns of each 16-column
  // block), experts e0 .. e0 + 7, tokens t0 + tg + 8 i (i < kTI).
  const int cs = lane >> 3, tg = lane & 7;
  float2 acc[kRsEB][kTI];
#pragma unroll
  for (int j = 0; j < kRsEB; ++j)
#pragma unroll
    for (int i = 0; i < kTI; ++i) acc[j][i] = make_float2(0.f, 0.f);
  int ok = 1;
  for (int q = 0; q < kRsSub; ++q) {
    // Every thread waits (bounded) for the sub-chunk; a timeout is reported
    // below and the rest of the CTA's work skipped.
    volatile int no_abort = 0;
    if (!mbar_wait(bar0 + 8 * q, 0, kRsWaitNs, &no_abort)) {
      ok = 0;
      break;
    }
    const int b_end = sub(q + 1) * (kRsChunk / 16);
#pragma unroll 2
    for (int blk = sub(q) * (kRsChunk / 16) + warp; blk < b_end; blk += kRsWarps) {
      const int col = blk * 16 + cs * 4;
      float4 w[kRsEB];
#pragma unroll
      for (int j = 0; j < kRsEB; ++j)
        w[j] = *reinterpret_cast<const float4 *>(Ws + static_cast<size_t>(j) * DS + col);
#pragma unroll
      for (int i = 0; i < kTI; ++i) {
        const uint2 xv = *reinterpret_cast<const uint2 *>(xs + static_cast<size_t>(tg + 8 * i) * xstride +
                                                          col * 2);
        const float2 xa = make_float2(bf16_lo(xv.x), bf16_hi(xv.x));
        const float2 xb = make_float2(bf16_lo(xv.y), bf16_hi(xv.y));
#pragma unroll
        for (int j = 0; j < kRsEB; ++j) {
          acc[j][i] = __ffma2_rn(xa, make_float2(w[j].x, w[j].y), acc[j][i]);
          acc[j][i] = __ffma2_rn(xb, make_float2(w[j].z, w[j].w), acc[j][i]);
        }
      }
    }
  }
  ok = __syncthreads_and(ok);
  if (threadIdx.x == 0) status[cta] = ok ? 0 : 1;
  if (!ok) return;  // reported; the copies were given a second to land

  // v[j * kTI + i]: this lane's column-set sum for expert j, token tg + 8 i.
  float v[V];
#pragma unroll
  for (int j = 0; j < kRsEB; ++j)
#pragma unroll
    for (int i = 0; i < kTI; ++i) v[j * kTI + i] = __fadd_rn(acc[j][i].x, acc[j][i].y);
  // Add the four column sets (lane bits 4 and 3) by a reduce-scatter: each
  // step the lane keeps the upper or lower half of its sums (by that bit)
  // and adds its partner's copy of them; lane (cs, tg) ends with sums
  // q0 .. q0 + V/4 - 1, q0 = (bit 4) V/2 + (bit 3) V/4.
#pragma unroll
  for (int step = 0; step < 2; ++step) {
    const int o = step == 0 ? 16 : 8, n = V >> (step + 1);
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int q = 0; q < n; ++q) {
      const float lo = v[q], hi = v[q + n];
      const float r = __shfl_xor_sync(0xffffffffu, up ? lo : hi, o);
      v[q] = __fadd_rn(up ? hi : lo, r);
    }
  }
  // The eight warps' sums, added in warp order (the W tile's space is free).
  __syncthreads();
  float *red = Ws;  // [warp][token TB][expert 8]
  {
    const int q0 = ((lane & 16) ? V / 2 : 0) + ((lane & 8) ? V / 4 : 0);
#pragma unroll
    for (int q = 0; q < V / 4; ++q) {
      const int jq = (q0 + q) / kTI, iq = (q0 + q) % kTI;
      red[(warp * TB + tg + 8 * iq) * kRsEB + jq] = v[q];
    }
  }
  __syncthreads();
  for (int o = threadIdx.x; o < TB * kRsEB; o += kRsThreads) {
    const int t = o / kRsEB, e = o % kRsEB;
    float sum = red[o];
#pragma unroll
    for (int w = 1; w < kRsWarps; ++w) sum = __fadd_rn(sum, red[w * TB * kRsEB + o]);
    if (t < nt && e < ne) h[(static_cast<size_t>(s) * B + t0 + t) * N + e0 + e] = sum;
  }
}

int rs_ti(int B) { return B <= 8 ? 1 : B <= 16 ? 2 : 4; }

}  // namespace

int router_split_count(int B, int N, int d, int n_sms) {
  const int nch = d / kRsChunk;
  const int blocks = ((N + kRsEB - 1) / kRsEB) * ((B + rs_tb(rs_ti(B)) - 1) / rs_tb(rs_ti(B)));
  const int need = (nch * kRsChunk + kRsMaxDS - 1) / kRsMaxDS;  // shared memory bound
  int S = n_sms / (blocks > 0 ? blocks : 1);
  if (S > kRsMaxSplits) S = kRsMaxSplits;
  if (S < need) S = need;
  if (S > nch) S = nch;
  return S < 1 ? 1 : S;
}

int router_split_ctas(int B, int N, int d, int n_sms) {
  const int TB = rs_tb(rs_ti(B));
  return ((N + kRsEB - 1) / kRsEB) * ((B + TB - 1) / TB) * router_split_count(B, N, d, n_sms);
}

namespace {

template <int kTI>
cudaError_t launch_rs(const uint16_t *x, const float *Wg, float *h, int B, int N, int d, int S,
                      int32_t *done, int32_t *status, cudaStream_t s) {
  const int nch = d / kRsChunk;
  const int DSmax = ((nch + S - 1) / S) * kRsChunk;
  const size_t smem = rs_smem_bytes(DSmax, rs_tb(kTI));
  cudaError_t e = cudaFuncSetAttribute(router_split_kernel<kTI>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid((N + kRsEB - 1) / kRsEB, S, (B + rs_tb(kTI) - 1) / rs_tb(kTI));
  return launch_pdl(router_split_kernel<kTI>, grid, dim3(kRsThreads), smem, s, x, Wg, h, B, N, d,
                    S, done, status);
}

}  // namespace

cudaError_t launch_router_split(const uint16_t *x, const float *Wg, float *h, int B, int N, int d,
                                int S, int32_t *done, int32_t *status, cudaStream_t s) {
  switch (rs_ti(B)) {
    case 1: return launch_rs<1>(x, Wg, h, B, N, d, S, done, status, s);
    case 2: return launch_rs<2>(x, Wg, h, B, N, d, S, done, status, s);
    default: return launch_rs<4>(x, Wg, h, B, N, d, S, done, status, s);
  }
}

}  // namespace xs
