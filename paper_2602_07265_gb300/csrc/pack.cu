// Packed expert weights: every 128-row x 64-column tile that the FFN kernels
// feed to the tensor cores, stored contiguously and already in the 128-byte
// swizzled shared-memory layout, so that one 1-D bulk copy brings a stage's
// weights in (a contiguous 16 or 32 KB block instead of 128 rows of 128 B
// spread over the matrix).
//
//   gate/up: block (e, mt, kk) = [gate tile | up tile], 32 KB, for expert e,
//            rows mt*128 .. +128 of F, columns kk*64 .. +64 of d;
//            blocks in (e, mt, kk) order.
//   down   : block (e, mt, kk) = one 16 KB tile, rows mt*128 of d, columns
//            kk*64 of F.
// Inside a tile, row r (0..127) takes bytes [r*128, r*128 + 128) and its
// 16-byte chunk c (columns c*8 .. +8) sits at chunk position c ^ (r % 8).
#include <cuda_runtime.h>

#include <cstdint>

#include "xs_internal.cuh"

namespace xs {
namespace {

constexpr int kRows = 128, kCols = 64, kTile = kRows * kCols * 2;

// W0 (and W1 if given) [n][M][K] bf16 -> P, `per` tiles per block (1 or 2).
__global__ void __launch_bounds__(256) pack_kernel(const uint4 *__restrict__ W0, const uint4 *__restrict__ W1,
                                                   uint8_t *__restrict__ P, int n, int M, int K) {
  pdl_wait();  // the weights may still be being written by the work before this call
  pdl_trigger();
  const int per = W1 ? 2 : 1;
  const int MT = M / kRows, KI = K / kCols, KC = K / 8;   // 16-byte chunks per row
  const long long chunks = static_cast<long long>(n) * M * KC;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < chunks * per;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int w = static_cast<int>(i / chunks);
    const long long j = i - w * chunks;
    const int cc = static_cast<int>(j % KC);
    const long long row = j / KC;                  // e * M + m
    const int e = static_cast<int>(row / M), m = static_cast<int>(row % M);
    const int mt = m / kRows, r = m % kRows, kk = cc / 8, c = cc % 8;
    const long long block = (static_cast<long long>(e) * MT + mt) * KI + kk;
    const long long dst = (block * per + w) * kTile + r * 128 + ((c ^ (r & 7)) << 4);
    const uint4 v = __ldg((w ? W1 : W0) + j);
    *reinterpret_cast<uint4 *>(P + dst) = v;
  }
}

}  // namespace

cudaError_t launch_pack(const uint16_t *W0, const uint16_t *W1, void *P, int n, int M, int K,
                        int n_sms, cudaStream_t s) {
  return launch_pdl(pack_kernel, dim3(n_sms * 8), dim3(256), 0, s, reinterpret_cast<const uint4 *>(W0),
                    reinterpret_cast<const uint4 *>(W1), static_cast<uint8_t *>(P), n, M, K);
}

}  // namespace xs
