// Router logits h = W_g x (step a1, Sec. 2.2) on the 5th-generation tensor
// cores, for batches large enough that fp32 FMA on the CUDA cores is the
// bound (2 B N d flops).
//
// fp32 accuracy from bf16 MMAs: every fp32 router weight w is the exact sum
// of three bf16 numbers, w1 = bf16(w), w2 = bf16(w - w1), w3 = bf16(w - w1 -
// w2) (each remainder is exact in fp32 and the last one has at most 8
// significant bits), and x is bf16 already, so each product x w_i is exact
// in fp32 and h = sum_k x_k (w1 + w2 + w3)_k is accumulated in fp32 in TMEM.
// The three planes are made in shared memory from the fp32 tile that TMA
// brings in, so W_g is read once per tile, as fp32.
//
// Tiling: the MMA's M = 128 rows are tokens (A = x, K-major, 128-byte
// swizzle, loaded by TMA), N = nt experts (B = the three weight planes,
// written by four converter warps in the same swizzled layout), K = 16 per
// instruction, 64 per pipeline stage.  An output tile of 128 tokens x nt
// experts is computed by a cluster of S <= 16 CTAs, each over 1/S of d; the CTAs
// park their fp32 partial tiles in shared memory and every CTA then adds up
// 128/S of the tile's rows from all S partials (distributed shared memory),
// in cluster-rank order, so h is reproducible bit for bit.
//
// Accuracy of the sum: the tensor cores' fp32 accumulation is not rounded
// to nearest at every addition, and over a long chain the error grows past
// what the fp32 CUDA-core sum gives.  So TMEM holds only one stage (64 of d,
// 12 MMAs) at a time: the accumulator restarts every stage and four drain
// warps add each stage's result to running sums in registers, one fp32
// round-to-nearest addition per stage, while the next stages are
// multiplied into up to seven other TMEM buffers.
//
// Roles (320 threads): warp 0 lane 0 issues TMA, warp 1 lane 0 issues the
// MMAs, warps 2-5 convert the weight planes, warps 6-9 drain the TMEM
// buffers.  Every mbarrier wait is bounded; every thread reaches both
// cluster barriers, so no CTA of a cluster can be left waiting on another.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cstring>

#include "tc_ptx.cuh"
#include "tmap.cuh"
#include "xs_internal.cuh"

namespace xs {
namespace {

using namespace ptx;

constexpr int kThreads = 320;
constexpr int kBM = 128;                       // tokens per tile (MMA M)
constexpr int kBK = 64;                        // K per stage
constexpr int kXBytes = kBM * kBK * 2;         // 16 KB of x per stage
constexpr int kMaxStages = 6;
constexpr int kAccBufs = 8;                    // TMEM accumulators in flight between MMA and drain
constexpr int kSmemBudget = 200 * 1024;        // stages (the partial tile reuses them)
constexpr uint64_t kWaitNs = 1000000000ull;    // 1 s per wait

struct RtParams {
  CUtensorMap tmX;     // x [B, d] bf16, box 64 x 128, 128-byte swizzle
  CUtensorMap tmW;     // W_g [N, d] fp32, box 64 x nt, no swizzle
  float *h;            // [B, N] out
  int32_t *done;       // [2] arrival counters of the selection kernels: zeroed here
  int32_t *status;     // [grid] per-CTA status, written by every CTA
  int B, N, d, tiles_n, stages;
};

__host__ __device__ constexpr int stage_bytes(int nt) { return kXBytes + nt * kBK * 4 + 3 * nt * 128; }

template <int kNt>
__global__ void __launch_bounds__(kThreads, 1) router_tc_kernel(const __grid_constant__ RtParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  constexpr int sb = stage_bytes(kNt);
  constexpr int kBufs = kAccBufs * kNt <= 256 ? kAccBufs : 256 / kNt;
  constexpr int kTmemCols = kBufs * kNt < 32 ? 32 : kBufs * kNt;
  const int stages = p.stages;
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + stages * sb;
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto conv_bar = [&](int s) { return bar0 + 8u * (kMaxStages + s); };
  auto empty_bar = [&](int s) { return bar0 + 8u * (2 * kMaxStages + s); };
  auto accf_bar = [&](int b) { return bar0 + 8u * (3 * kMaxStages + b); };
  auto acce_bar = [&](int b) { return bar0 + 8u * (3 * kMaxStages + kAccBufs + b); };
  const uint32_t drain_bar = bar0 + 8u * (3 * kMaxStages + 2 * kAccBufs);
  uint32_t *tmem_slot =
      reinterpret_cast<uint32_t *>(smem + stages * sb + 8 * (3 * kMaxStages + 2 * kAccBufs + 1));
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  auto x_s = [&](int s) { return sbase + s * sb; };
  auto w_s = [&](int s) { return smem + s * sb + kXBytes; };
  auto plane_s = [&](int s, int pl) { return sbase + s * sb + kXBytes + kNt * kBK * 4 + pl * kNt * 128; };

  pdl_wait();
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = static_cast<int>(cluster_nctarank());
  const int split = static_cast<int>(cluster_ctarank());
  const int tile = blockIdx.x / S;
  const int m0 = (tile / p.tiles_n) * kBM, n0 = (tile % p.tiles_n) * kNt;
  const int KI = p.d / kBK;
  const int k_begin = KI * split / S, k_end = KI * (split + 1) / S;

  if (threadIdx.x == 0) {
    if (blockIdx.x == 0) {
      p.done[0] = 0;
      p.done[1] = 0;
      p.done[2] = 0;
      p.done[3] = 0;
    }
    for (int s = 0; s < kMaxStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(conv_bar(s), 128);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < kBufs; ++b) {
      mbar_init(accf_bar(b), 1);
      mbar_init(acce_bar(b), 128);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&p.tmX);
    prefetch_tmap(&p.tmW);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_last();  // W_g and x are reread by other tiles
      const uint32_t tx = kXBytes + kNt * kBK * 4;
      int stage = 0;
      uint32_t phase = 0, issued_mask = 0, issued_phase = 0;
      for (int kk = k_begin; kk < k_end; ++kk) {
        if (!mbar_wait(empty_bar(stage), phase ^ 1u, kWaitNs, abort_flag)) {
          *abort_flag = 1;
          break;
        }
        mbar_arrive_expect_tx(full_bar(stage), tx);
        tma_load_2d(x_s(stage), &p.tmX, full_bar(stage), kk * kBK, m0, pol);
        tma_load_2d(smem_u32(w_s(stage)), &p.tmW, full_bar(stage), kk * kBK, n0, pol);
        issued_mask |= 1u << stage;
        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
        if (++stage == stages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      // Never leave with copies in flight: wait (bounded) for the last load of every stage.
      volatile int no_abort = 0;
      for (int s = 0; s < stages; ++s)
        if ((issued_mask >> s) & 1u) mbar_wait(full_bar(s), (issued_phase >> s) & 1u, kWaitNs, &no_abort);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(kBM, kNt);
      int stage = 0;
      uint32_t phase = 0;
      bool any = false;
      for (int kk = k_begin; kk < k_end; ++kk) {
        const int i = kk - k_begin, buf = i % kBufs;
        const uint32_t use = static_cast<uint32_t>(i / kBufs);
        if (!mbar_wait(conv_bar(stage), phase, kWaitNs, abort_flag) ||
            !mbar_wait(acce_bar(buf), (use & 1u) ^ 1u, kWaitNs, abort_flag)) {
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d0 = tmem + static_cast<uint32_t>(buf * kNt);
#pragma unroll
        for (int ks = 0; ks < kBK / 16; ++ks) {
          const uint64_t da = sw128_desc(x_s(stage) + ks * 32);
#pragma unroll
          for (int pl = 0; pl < 3; ++pl)
            mma_bf16(d0, da, sw128_desc(plane_s(stage, pl) + ks * 32), idesc,
                     (ks > 0 || pl > 0) ? 1u : 0u);
        }
        any = true;
        mma_commit(empty_bar(stage));
        mma_commit(accf_bar(buf));
        if (++stage == stages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (any) {  // all issued MMAs done before TMEM is released
        volatile int no_abort = 0;
        mma_commit(drain_bar);
        mbar_wait(drain_bar, 0, kWaitNs, &no_abort);
      }
    }
  } else if (warp < 6) {
    // ------------------------------------------------ weight planes
    const int cw = warp - 2;
    int stage = 0;
    uint32_t phase = 0;
    for (int kk = k_begin; kk < k_end; ++kk) {
      if (!mbar_wait(full_bar(stage), phase, kWaitNs, abort_flag)) {
        *abort_flag = 1;
        break;
      }
      const float *wt = reinterpret_cast<const float *>(w_s(stage));
#pragma unroll
      for (int r = cw; r < kNt; r += 4) {
        const float2 v = *reinterpret_cast<const float2 *>(wt + r * kBK + 2 * lane);
        const __nv_bfloat162 a1 = __floats2bfloat162_rn(v.x, v.y);
        const float2 f1 = __bfloat1622float2(a1);
        const float rx = v.x - f1.x, ry = v.y - f1.y;
        const __nv_bfloat162 a2 = __floats2bfloat162_rn(rx, ry);
        const float2 f2 = __bfloat1622float2(a2);
        const __nv_bfloat162 a3 = __floats2bfloat162_rn(rx - f2.x, ry - f2.y);
        // bf16 columns 2 lane, 2 lane + 1: 16-byte chunk lane / 4 of row r,
        // stored at chunk (lane / 4) ^ (r % 8) as the 128-byte swizzle lays out.
        const uint32_t off = r * 128 + ((((lane >> 2) ^ (r & 7)) << 4) | ((lane & 3) << 2));
        asm volatile("st.shared.b32 [%0], %1;" ::"r"(plane_s(stage, 0) + off),
                     "r"(*reinterpret_cast<const uint32_t *>(&a1)) : "memory");
        asm volatile("st.shared.b32 [%0], %1;" ::"r"(plane_s(stage, 1) + off),
                     "r"(*reinterpret_cast<const uint32_t *>(&a2)) : "memory");
        asm volatile("st.shared.b32 [%0], %1;" ::"r"(plane_s(stage, 2) + off),
                     "r"(*reinterpret_cast<const uint32_t *>(&a3)) : "memory");
      }
      fence_proxy_async_smem();
      mbar_arrive(conv_bar(stage));
      if (++stage == stages) {
        stage = 0;
        phase ^= 1u;
      }
    }
  } else {
    // ------------------------------------------------ drain: one fp32 add per stage
    const int q = warp & 3, row = q * 32 + lane;
    float sum[kNt];
#pragma unroll
    for (int j = 0; j < kNt; ++j) sum[j] = 0.f;
    for (int kk = k_begin; kk < k_end; ++kk) {
      const int i = kk - k_begin, buf = i % kBufs;
      const uint32_t use = static_cast<uint32_t>(i / kBufs);
      if (!mbar_wait(accf_bar(buf), use & 1u, kWaitNs, abort_flag)) {
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      const uint32_t ta = tmem + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(buf * kNt);
#pragma unroll
      for (int c0 = 0; c0 < kNt; c0 += 16) {
        float v[16];
        tmem_ld16(ta + c0, v);
#pragma unroll
        for (int j = 0; j < 16; ++j) sum[c0 + j] = __fadd_rn(sum[c0 + j], v[j]);
      }
      tc_fence_before();
      mbar_arrive(acce_bar(buf));
    }
    // Every load was consumed by an MMA that has completed: the stages are
    // idle and hold the partial tile [128][nt + 4] fp32 now.
    float *part = reinterpret_cast<float *>(smem) + row * (kNt + 4);
#pragma unroll
    for (int j = 0; j < kNt; j += 4)
      *reinterpret_cast<float4 *>(part + j) = make_float4(sum[j], sum[j + 1], sum[j + 2], sum[j + 3]);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  cluster_sync();  // every CTA's partial tile is in its shared memory

  // Rows [split * 128 / S, (split + 1) * 128 / S) of the tile, summed over
  // the S partials in rank order.
  const int rows = kBM / S, r_begin = split * rows;
  for (int e = threadIdx.x; e < rows * kNt; e += kThreads) {
    const int r = r_begin + e / kNt, c = e % kNt;
    const int t = m0 + r, j = n0 + c;
    const uint32_t a = sbase + static_cast<uint32_t>((r * (kNt + 4) + c) * 4);
    float part[16];  // all remote loads in flight first, then the sum in rank order
#pragma unroll
    for (int src = 0; src < 16; ++src)
      part[src] = src < S ? ld_cluster_f32(a, static_cast<uint32_t>(src)) : 0.f;
    float v = 0.f;
#pragma unroll
    for (int src = 0; src < 16; ++src)
      if (src < S) v = __fadd_rn(v, part[src]);
    if (t < p.B && j < p.N) p.h[static_cast<size_t>(t) * p.N + j] = v;
  }
  cluster_sync();  // no CTA leaves while another still reads its shared memory
  if (threadIdx.x == 0) p.status[blockIdx.x] = *abort_flag ? XS_DEV_TIMEOUT : XS_DEV_OK;
}

struct RtShape {
  int nt, S, tiles_n, grid, stages;
};

int stages_for(int nt) {
  const int st = kSmemBudget / stage_bytes(nt);
  return st > kMaxStages ? kMaxStages : st;
}

size_t smem_for(int nt) {
  return static_cast<size_t>(stages_for(nt)) * stage_bytes(nt) +
         8 * (3 * kMaxStages + 2 * kAccBufs + 1) + 16 + 1024;
}

using KernelFn = void (*)(RtParams);

KernelFn kernel_for(int nt) {
  return nt == 16 ? router_tc_kernel<16> : nt == 32 ? router_tc_kernel<32> : router_tc_kernel<64>;
}

// Clusters of S CTAs of the nt variant that the current device can hold at
// once (cached per device; host threads that race on it store the same
// value); 0 if the query fails.
int cluster_cap(int nt, int S) {
  constexpr int kDevs = 64;
  static std::atomic<int> cache[kDevs][3][5];  // the count + 1, 0 while unknown
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kDevs) return 0;
  const int a = nt == 16 ? 0 : nt == 32 ? 1 : 2;
  const int b = S == 1 ? 0 : S == 2 ? 1 : S == 4 ? 2 : S == 8 ? 3 : 4;
  const int known = cache[dev][a][b].load(std::memory_order_relaxed);
  if (known > 0) return known - 1;
  int n = 0;
  const KernelFn k = kernel_for(nt);
  if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem_for(nt))) == cudaSuccess &&
      cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(S);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem_for(nt);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, k, &cfg) != cudaSuccess) n = 0;
  }
  cudaGetLastError();  // a failed query leaves no sticky error
  cache[dev][a][b].store(n + 1, std::memory_order_relaxed);
  return n;
}

// Experts per tile (nt) and CTAs per cluster (S).  A CTA's time is a fixed
// part (first loads, pipeline drain, cluster barriers, reduction: about
// 6 us) plus about 0.55 us per K step of 64 whatever nt is (the round trip
// of a stage through TMA, plane conversion and MMA), so the shape with the
// fewest K steps per CTA wins, among those whose clusters the device runs
// at once; then the larger grid, then the fewer bytes per CTA.
RtShape choose_shape(int B, int N, int d, int n_sms) {
  const int tiles_m = (B + kBM - 1) / kBM, KI = d / kBK;
  RtShape best = {64, 1, (N + 63) / 64, 0, 0};
  double best_cost = 0.0;
  long long best_bytes = -1;
  for (int nt : {64, 32, 16}) {
    const int tn = (N + nt - 1) / nt;
    for (int S : {16, 8, 4, 2, 1}) {
      if (S > KI) continue;
      const int grid = tiles_m * tn * S;
      if (grid > n_sms || tiles_m * tn > cluster_cap(nt, S)) continue;
      const int steps = (KI + S - 1) / S;
      const double cost = static_cast<double>(steps);
      const long long bytes = static_cast<long long>(steps) * (kXBytes + nt * kBK * 4);
      const bool better = best.grid == 0 || cost < best_cost ||
                          (cost == best_cost && (grid > best.grid ||
                                                 (grid == best.grid && bytes < best_bytes)));
      if (better) {
        best = {nt, S, tn, grid, 0};
        best_cost = cost;
        best_bytes = bytes;
      }
    }
  }
  if (best.grid == 0) best = {64, 1, (N + 63) / 64, tiles_m * ((N + 63) / 64), 0};
  best.stages = stages_for(best.nt);
  return best;
}

}  // namespace

int router_tc_ctas(int B, int N, int d, int n_sms) {
  (void)d;
  (void)n_sms;
  return ((B + kBM - 1) / kBM) * ((N + 15) / 16) * 16;  // bound on the grid of every shape
}

cudaError_t launch_router_tc(const uint16_t *x, const float *Wg, float *h, int B, int N, int d,
                             int32_t *done, int32_t *status, int n_sms, int *grid_out,
                             cudaStream_t s) {
  const RtShape sh = choose_shape(B, N, d, n_sms);
  *grid_out = sh.grid;
  RtParams p;
  memset(&p, 0, sizeof(p));
  if (!encode_tmap_2d(&p.tmX, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, x, d, B, kBK, kBM,
                      CU_TENSOR_MAP_SWIZZLE_128B) ||
      !encode_tmap_2d(&p.tmW, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, Wg, d, N, kBK, sh.nt,
                      CU_TENSOR_MAP_SWIZZLE_NONE))
    return cudaErrorInvalidValue;
  p.h = h;
  p.done = done;
  p.status = status;
  p.B = B;
  p.N = N;
  p.d = d;
  p.tiles_n = sh.tiles_n;
  p.stages = sh.stages;
  const KernelFn kern = kernel_for(sh.nt);
  const size_t smem = smem_for(sh.nt);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(sh.grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = sh.S;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, p);
}

}  // namespace xs
