// Expert SwiGLU FFN over the routed pairs (step a8), plain CUDA-core version.
//
// Phase 1: act[r, f] = silu(W_gate[e, f] . xp[r]) * (W_up[e, f] . xp[r]) (bf16)
// Phase 2: out[r, c] = W_down[e, c] . act[r]                              (fp32)
// for every row r of a tile of expert e (Sec. 2.1: E_e(x)).  One warp owns one
// weight row and walks the tile's tokens in groups of 8, so each weight row is
// read once per 8 tokens.
#include <cuda_bf16.h>

#include "xs_internal.cuh"

namespace xs {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kTokGroup = 8;
constexpr int kRowsPerBlock = 8;

__device__ __forceinline__ void unpack8(const uint4 v, float f[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}

__device__ __forceinline__ float silu(float g) { return g / (1.f + expf(-g)); }

__global__ void __launch_bounds__(256) gateup_simt_kernel(FfnArgs a) {
  const int ti = blockIdx.y;
  if (ti >= a.meta->n_tiles) return;
  const Tile tl = a.tiles[ti];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int f = blockIdx.x * kRowsPerBlock + warp;
  if (f >= a.F) return;
  const int d = a.d;
  const uint16_t *wg = a.W_gate + ((size_t)tl.expert * a.F + f) * d;
  const uint16_t *wu = a.W_up + ((size_t)tl.expert * a.F + f) * d;
  for (int j0 = 0; j0 < tl.ntok; j0 += kTokGroup) {
    float ag[kTokGroup], au[kTokGroup];
#pragma unroll
    for (int j = 0; j < kTokGroup; ++j) ag[j] = au[j] = 0.f;
    for (int c = lane * 8; c < d; c += 256) {
      float gw[8], uw[8];
      unpack8(__ldg(reinterpret_cast<const uint4 *>(wg + c)), gw);
      unpack8(__ldg(reinterpret_cast<const uint4 *>(wu + c)), uw);
#pragma unroll
      for (int j = 0; j < kTokGroup; ++j) {
        if (j0 + j < tl.ntok) {
          float xv[8];
          unpack8(__ldg(reinterpret_cast<const uint4 *>(a.xp + (size_t)(tl.row0 + j0 + j) * d + c)), xv);
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            ag[j] = fmaf(xv[q], gw[q], ag[j]);
            au[j] = fmaf(xv[q], uw[q], au[j]);
          }
        }
      }
    }
#pragma unroll
    for (int j = 0; j < kTokGroup; ++j)
#pragma unroll
      for (int o = 16; o; o >>= 1) {
        ag[j] += __shfl_xor_sync(kFull, ag[j], o);
        au[j] += __shfl_xor_sync(kFull, au[j], o);
      }
    float g = 0.f, u = 0.f;
#pragma unroll
    for (int j = 0; j < kTokGroup; ++j)
      if (lane == j) {
        g = ag[j];
        u = au[j];
      }
    if (lane < kTokGroup && j0 + lane < tl.ntok) {
      const __nv_bfloat16 v = __float2bfloat16_rn(silu(g) * u);
      a.act[(size_t)(tl.row0 + j0 + lane) * a.F + f] = *reinterpret_cast<const uint16_t *>(&v);
    }
  }
}

__global__ void __launch_bounds__(256) down_simt_kernel(FfnArgs a) {
  const int ti = blockIdx.y;
  if (ti >= a.meta->n_tiles) return;
  const Tile tl = a.tiles[ti];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int c = blockIdx.x * kRowsPerBlock + warp;
  if (c >= a.d) return;
  const int F = a.F;
  const uint16_t *wd = a.W_down + ((size_t)tl.expert * a.d + c) * F;
  for (int j0 = 0; j0 < tl.ntok; j0 += kTokGroup) {
    float ao[kTokGroup];
#pragma unroll
    for (int j = 0; j < kTokGroup; ++j) ao[j] = 0.f;
    for (int f = lane * 8; f < F; f += 256) {
      float dw[8];
      unpack8(__ldg(reinterpret_cast<const uint4 *>(wd + f)), dw);
#pragma unroll
      for (int j = 0; j < kTokGroup; ++j) {
        if (j0 + j < tl.ntok) {
          float av[8];
          unpack8(*reinterpret_cast<const uint4 *>(a.act + (size_t)(tl.row0 + j0 + j) * F + f), av);
#pragma unroll
          for (int q = 0; q < 8; ++q) ao[j] = fmaf(av[q], dw[q], ao[j]);
        }
      }
    }
#pragma unroll
    for (int j = 0; j < kTokGroup; ++j)
#pragma unroll
      for (int o = 16; o; o >>= 1) ao[j] += __shfl_xor_sync(kFull, ao[j], o);
    float o = 0.f;
#pragma unroll
    for (int j = 0; j < kTokGroup; ++j)
      if (lane == j) o = ao[j];
    if (lane < kTokGroup && j0 + lane < tl.ntok) a.out[(size_t)(tl.row0 + j0 + lane) * a.d + c] = o;
  }
}

}  // namespace

size_t ffn_part_bytes(int n_sms) { return 256; }
size_t ffn_cnt_words(int max_tiles, int d, int F) { return 64; }

cudaError_t launch_ffn_gate_up(const FfnArgs &a, cudaStream_t s) {
  dim3 grid((a.F + kRowsPerBlock - 1) / kRowsPerBlock, a.max_tiles);
  gateup_simt_kernel<<<grid, 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_ffn_down(const FfnArgs &a, cudaStream_t s) {
  dim3 grid((a.d + kRowsPerBlock - 1) / kRowsPerBlock, a.max_tiles);
  down_simt_kernel<<<grid, 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace xs
