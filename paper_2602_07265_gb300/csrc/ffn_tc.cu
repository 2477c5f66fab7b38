// Expert SwiGLU FFN over the routed pairs (step a8) on the 5th-generation
// tensor cores: tcgen05.mma with TMEM accumulators, operands fed by TMA.
//
//   gate/up phase: act[r, f] = silu(W_gate[e, f] . xp[r]) * (W_up[e, f] . xp[r])   (bf16)
//   down phase   : out[r, c] = W_down[e, c] . act[r]                                (fp32)
// for every routed pair row r of expert e (Sec. 2.1: E_e(x)).
//
// Decode batches give each expert a handful of tokens, so the layer streams
// the used experts' weights once and is bound by HBM.  The weights fill the
// MMA's M = 128 dimension ("swap AB") and the expert's tokens are the N
// dimension (16..128, a multiple of 16, chosen per tile at run time).
//
// Work split ("stream-K"): a unit is (tile of <= 128 tokens of one expert,
// 128 weight rows); its K loop has K/64 steps.  The units' steps are laid end
// to end and cut into equal contiguous ranges, one per CTA, so every SM
// streams the same number of weight bytes.  A unit cut between CTAs is
// finished by whichever CTA arrives last: every piece writes its fp32 partial
// accumulator, bumps the unit's counter, and the last one adds the pieces in
// K order (deterministic) and runs the epilogue.  No CTA ever waits for
// another.
//
// Roles inside a CTA (192 threads): warp 0 lane 0 issues TMA loads into a
// ring of shared-memory stages; warp 1 lane 0 issues the MMAs into one of two
// TMEM accumulator buffers; warps 2-5 (one TMEM lane quarter each) drain the
// accumulators.  Every mbarrier wait is bounded in time.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstring>

#include "tc_ptx.cuh"
#include "tmap.cuh"
#include "xs_internal.cuh"

namespace xs {
namespace {

using namespace ptx;

constexpr int kBM = 128;          // weight rows per unit (MMA M)
constexpr int kBK = 64;           // bf16 per K step (one 128-byte swizzle row)
constexpr int kBoxTok = 16;       // token rows per TMA box of the B operand
constexpr int kThreads = 192;
constexpr int kEpiThreads = 128;
constexpr int kTileBytes = kBM * kBK * 2;     // 16 KB
constexpr uint64_t kWaitNs = 1000000000ull;   // 1 s per wait

template <bool kGateUp>
struct Cfg {
  static constexpr int kNumA = kGateUp ? 2 : 1;          // weight tiles per stage
  static constexpr int kStages = kGateUp ? 3 : 6;   // measured best on GB300 (3, 4 and 2; 4, 5 and 6)
  static constexpr int kStageBytes = kNumA * kTileBytes + kTileBytes;
  // Weights fetched before pdl_wait(): the ring's first stages, then an L2
  // prefetch of the weights after them, 64 KB per CTA (measured best on GB300
  // among 0 to 256 KB; more competes with the kernel before for HBM).
  static constexpr int kL2Prefetch = 64 * 1024;
  static constexpr int kAccCols = kGateUp ? 256 : 128;   // TMEM columns per buffer
  static constexpr int kTmemCols = 2 * kAccCols;
  static constexpr int kBarOffset = kStages * kStageBytes;
  static constexpr int kSmemBytes = kBarOffset + 256 + 1024;  // + barriers + alignment slack
};

struct TcParams {
  CUtensorMap tmA0;     // W_gate (gate/up) or W_down (down): [N * M, K] bf16, box 128 x 64
  CUtensorMap tmA1;     // W_up (gate/up only)
  CUtensorMap tmS0;     // the same for the shared experts (experts >= n_routed)
  CUtensorMap tmS1;
  CUtensorMap tmB[4];   // xp (gate/up) or act (down): [max_rows, K] bf16, boxes of
                        // 16, 32, 64, 128 rows x 64
  const uint8_t *pk;        // nullable: packed weights (pack.cu); then tmA0 / tmA1 are unused
  const uint8_t *pk_shared; // packed shared experts
  const Tile *tiles;
  Meta *meta;
  xs_stats *stats;
  float *part;          // [grid][2 slots][kNumA][128 cols][128 lanes] fp32
  int32_t *cnt;         // [units] arrival counters, zeroed by the routing kernel
  uint16_t *act_out;    // gate/up output [max_rows, M]
  float *out;           // down output [max_rows, M]
  int M;                // weight rows per expert: F (gate/up) or d (down)
  int K;                // reduction length: d (gate/up) or F (down)
  int grid;
  int n_routed;         // N: tiles of experts >= N use tmS0 / tmS1
  int has_shared;
  int expert_base;      // routed expert e uses weights e - expert_base (expert parallelism)
};

// The FFN work of the call (Meta): routed tiles [t0, t1) then shared tiles
// [s0, s1); work tile i is tile tile(i).
struct WorkTiles {
  int t0, n_routed, s0, n;
  __device__ int tile(int i) const { return i < n_routed ? t0 + i : s0 + (i - n_routed); }
};

__device__ __forceinline__ WorkTiles work_tiles(const Meta *m) {
  WorkTiles w;
  w.t0 = __ldcg(&m->ffn_t0);
  w.n_routed = __ldcg(&m->ffn_t1) - w.t0;
  w.s0 = __ldcg(&m->ffn_s0);
  w.n = w.n_routed + (__ldcg(&m->ffn_s1) - w.s0);
  return w;
}

struct Range {
  long long I;      // total K steps
  int G;            // CTAs that take part
  int KI;           // K steps per unit
  __device__ long long begin(int c) const { return I * c / G; }
  // CTA whose range holds step i.
  __device__ int cta_of(long long i) const {
    int c = static_cast<int>((i * G) / I);
    while (c + 1 < G && begin(c + 1) <= i) ++c;
    while (c > 0 && begin(c) > i) --c;
    return c;
  }
  // Partial slot a CTA uses for unit u: 0 for the unit its range starts in, 1 otherwise.
  __device__ int slot(int c, long long u) const { return (begin(c) / KI == u) ? 0 : 1; }
};

__device__ __forceinline__ void set_status(const TcParams &p, int code) {
  atomicMax(&p.meta->status, code);
  if (p.stats) atomicMax(&p.stats->status, code);
}

__device__ __forceinline__ float silu(float g) { return g / (1.f + expf(-g)); }

template <bool kGateUp>
__global__ void __launch_bounds__(kThreads, 1) ffn_tc_kernel(const __grid_constant__ TcParams p) {
  using C = Cfg<kGateUp>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + C::kBarOffset;
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (C::kStages + s); };
  auto accfull_bar = [&](int b) { return bar0 + 8u * (2 * C::kStages + b); };
  auto accempty_bar = [&](int b) { return bar0 + 8u * (2 * C::kStages + 2 + b); };
  const uint32_t drain_bar = bar0 + 8u * (2 * C::kStages + 4);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + C::kBarOffset + 8 * (2 * C::kStages + 5));
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  volatile int *s_flag = reinterpret_cast<volatile int *>(tmem_slot + 2);

  // The routing kernels that wrote meta and tiles finished before this grid
  // could start (every kernel of the chain calls pdl_trigger() only after its
  // own pdl_wait()), so they may be read here through L2 before pdl_wait();
  // only the token operand and the outputs depend on the kernel just before.
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const WorkTiles wt = work_tiles(p.meta);
  const int n_tiles = wt.n;
  const int MT = p.M / kBM, KI = p.K / kBK;
  Range rg;
  rg.KI = KI;
  rg.I = static_cast<long long>(n_tiles) * MT * KI;
  rg.G = ffn_ctas(static_cast<long long>(n_tiles) * MT, KI, p.grid);
  if (rg.I == 0 || static_cast<int>(blockIdx.x) >= rg.G) {
    pdl_wait();
    pdl_trigger();
    return;
  }
  const int cta = blockIdx.x;
  const long long it_begin = rg.begin(cta), it_end = rg.begin(cta + 1);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(accfull_bar(b), 1);
      mbar_init(accempty_bar(b), 1);
    }
    mbar_init(drain_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
    if (p.pk == nullptr) {
      prefetch_tmap(&p.tmA0);
      if (kGateUp) prefetch_tmap(&p.tmA1);
      if (p.has_shared) {
        prefetch_tmap(&p.tmS0);
        if (kGateUp) prefetch_tmap(&p.tmS1);
      }
    }
    for (int i = 0; i < 4; ++i) prefetch_tmap(&p.tmB[i]);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Where unit u's operands come from.
  struct Src {
    int ntok, row0, bsel, arow;
    uint32_t tx;
    const CUtensorMap *mA0, *mA1;
    const uint8_t *pblk;   // packed: the unit's blocks are consecutive, one per K step
  };
  // Before pdl_wait() the tile is read through L2 only; after it, with a
  // plain load that also leaves it in L1 for the MMA and epilogue warps.
  auto src_of = [&](long long u, bool early) {
    const int4 *tp = reinterpret_cast<const int4 *>(p.tiles) + wt.tile(static_cast<int>(u / MT));
    const int4 t4 = early ? __ldcg(tp) : *tp;
    Src r;
    r.ntok = t4.z;
    r.row0 = t4.y;
    const int mt = static_cast<int>(u % MT);
    // One box of 16, 32, 64 or 128 token rows covers the tile's tokens.
    r.bsel = r.ntok <= 16 ? 0 : r.ntok <= 32 ? 1 : r.ntok <= 64 ? 2 : 3;
    r.tx = C::kNumA * kTileBytes + (kBoxTok << r.bsel) * kBK * 2;
    const bool routed = t4.x < p.n_routed;
    r.mA0 = routed ? &p.tmA0 : &p.tmS0;
    r.mA1 = routed ? &p.tmA1 : &p.tmS1;
    const int e_local = routed ? t4.x - p.expert_base : t4.x - p.n_routed;
    r.arow = e_local * p.M + mt * kBM;
    r.pblk = p.pk ? (routed ? p.pk : p.pk_shared) +
                        ((static_cast<size_t>(e_local) * MT + mt) * KI) * (C::kNumA * kTileBytes)
                  : nullptr;
    return r;
  };
  auto load_weights = [&](const Src &r, int kk, uint32_t sA, uint32_t bar, uint64_t pol) {
    if (r.pblk) {
      bulk_load(sA, r.pblk + static_cast<size_t>(kk) * (C::kNumA * kTileBytes), C::kNumA * kTileBytes,
                bar, pol);
    } else {
      tma_load_2d(sA, r.mA0, bar, kk * kBK, r.arow, pol);
      if (kGateUp) tma_load_2d(sA + kTileBytes, r.mA1, bar, kk * kBK, r.arow, pol);
    }
  };
  const bool producer = warp == 0 && lane == 0;
  const int n_pre = (it_end - it_begin) < C::kStages ? static_cast<int>(it_end - it_begin) : C::kStages;
  // The CTA's steps as segments (unit u, steps [k0, k1) of it), in the order
  // all three roles process them: first the piece of the last unit that the
  // next CTA finishes, then the piece of the first unit that the previous
  // CTA began, then the whole units between.  Both pieces of every unit cut
  // between two CTAs are then done early, so their partial sums are added
  // early too, and a CTA ends on a whole unit (whose epilogue is one TMEM
  // drain) instead of a cut one (partial store, fence, arrival, the other
  // pieces' loads).  Results do not depend on the order: the pieces are
  // added in CTA order.
  struct Seg {
    long long u;
    int k0, k1;
  };
  const long long u_first = it_begin / KI, u_last = (it_end - 1) / KI;
  const int kT0 = static_cast<int>(it_begin - u_first * KI);  // the first unit starts here
  const int kH1 = static_cast<int>(it_end - u_last * KI);     // the last unit ends here
  const bool one_unit = u_first == u_last;
  const int nH = (!one_unit && kH1 < KI) ? 1 : 0, nT = (!one_unit && kT0 > 0) ? 1 : 0;
  const long long fu0 = u_first + nT;                          // first whole unit
  const int n_seg = one_unit ? 1 : nH + nT + static_cast<int>(u_last - nH - fu0 + 1);
  auto seg_at = [&](int i) -> Seg {
    if (one_unit) return Seg{u_first, kT0, kH1};
    if (i < nH) return Seg{u_last, 0, kH1};
    if (i < nH + nT) return Seg{u_first, kT0, KI};
    return Seg{fu0 + (i - nH - nT), 0, KI};
  };
  // The producer walks its K steps with a cursor (segment si: unit u, step
  // kk of [.., k1)) and re-reads the unit's source only when u changes.
  struct Cursor {
    int si;
    long long u;
    int kk, k1;
    bool fresh;
  };
  const Seg s0 = seg_at(0);
  const Cursor c_begin{0, s0.u, s0.k0, s0.k1, true};
  auto advance = [&](Cursor &c) {
    if (++c.kk == c.k1) {
      if (++c.si < n_seg) {
        const Seg g = seg_at(c.si);
        c.u = g.u;
        c.kk = g.k0;
        c.k1 = g.k1;
      }
      c.fresh = true;
    }
  };
  auto source = [&](Cursor &c, Src &r, bool early) {
    if (c.fresh) {
      r = src_of(c.u, early);
      c.fresh = false;
    }
  };
  uint64_t pol_w = 0, pol_x = 0;
  if (producer) {
    // Every stage is free at the start: fill the ring with weights and warm L2
    // with the weights that follow.
    pol_w = policy_evict_first();
    pol_x = policy_evict_last();
    Cursor c = c_begin;
    Src r{};
    for (int i = 0; i < n_pre; ++i, advance(c)) {
      source(c, r, true);
      mbar_arrive_expect_tx(full_bar(i), r.tx);
      load_weights(r, c.kk, sbase + i * C::kStageBytes, full_bar(i), pol_w);
    }
    if (p.pk) {
      const long long n_pf = C::kL2Prefetch / (C::kNumA * kTileBytes);
      for (long long it = it_begin + n_pre; it < it_end && it < it_begin + n_pre + n_pf; ++it, advance(c)) {
        source(c, r, true);
        bulk_prefetch_l2(r.pblk + static_cast<size_t>(c.kk) * (C::kNumA * kTileBytes),
                         C::kNumA * kTileBytes);
      }
    }
  }
  pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    if (lane == 0) {
      uint32_t issued_mask = 0, issued_phase = 0;
      Cursor c = c_begin;
      Src r{};
      // Token operand of the stages filled above.
      for (int i = 0; i < n_pre; ++i, advance(c)) {
        source(c, r, false);
        tma_load_2d(sbase + i * C::kStageBytes + C::kNumA * kTileBytes, &p.tmB[r.bsel], full_bar(i),
                    c.kk * kBK, r.row0, pol_x);
        issued_mask |= 1u << i;
      }
      int stage = static_cast<int>(n_pre % C::kStages);
      uint32_t phase = n_pre == C::kStages ? 1u : 0u;
      bool ok = true;
      for (long long it = it_begin + n_pre; it < it_end; ++it, advance(c)) {
        source(c, r, false);
        const int kk = c.kk;
        if (!mbar_wait(empty_bar(stage), phase ^ 1u, kWaitNs, abort_flag)) {
          ok = false;
          break;
        }
        const uint32_t sA = sbase + stage * C::kStageBytes;
        mbar_arrive_expect_tx(full_bar(stage), r.tx);
        load_weights(r, kk, sA, full_bar(stage), pol_w);
        tma_load_2d(sA + C::kNumA * kTileBytes, &p.tmB[r.bsel], full_bar(stage), kk * kBK, r.row0, pol_x);
        issued_mask |= 1u << stage;
        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
        if (++stage == C::kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) {
        set_status(p, XS_DEV_TIMEOUT);
        *abort_flag = 1;
      }
      // Never leave with copies in flight: wait (bounded) for the last load of every stage.
      volatile int no_abort = 0;
      for (int s = 0; s < C::kStages; ++s)
        if ((issued_mask >> s) & 1u) mbar_wait(full_bar(s), (issued_phase >> s) & 1u, kWaitNs, &no_abort);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int segi = 0;
      bool ok = true, any = false;
      for (; ok && segi < n_seg; ++segi) {
        const Seg g = seg_at(segi);
        const long long u = g.u;
        const int k0 = g.k0, k1 = g.k1;
        const Tile tl = p.tiles[wt.tile(static_cast<int>(u / MT))];
        const int n_mma = ((tl.ntok + 15) / 16) * 16;
        const uint32_t idesc = idesc_bf16(kBM, n_mma);
        const int buf = segi & 1;
        const uint32_t use = static_cast<uint32_t>(segi >> 1);
        if (!mbar_wait(accempty_bar(buf), (use & 1u) ^ 1u, kWaitNs, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d0 = tmem + buf * C::kAccCols;
        for (int kk = k0; kk < k1; ++kk) {
          if (!mbar_wait(full_bar(stage), phase, kWaitNs, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sA = sbase + stage * C::kStageBytes;
          const uint32_t sB = sA + C::kNumA * kTileBytes;
#pragma unroll
          for (int ks = 0; ks < kBK / 16; ++ks) {
            const uint32_t acc = (kk > k0 || ks > 0) ? 1u : 0u;
            const uint64_t db = sw128_desc(sB + ks * 32);
            mma_bf16(d0, sw128_desc(sA + ks * 32), db, idesc, acc);
            if (kGateUp) mma_bf16(d0 + 128, sw128_desc(sA + kTileBytes + ks * 32), db, idesc, acc);
          }
          any = true;
          mma_commit(empty_bar(stage));
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        mma_commit(accfull_bar(buf));
      }
      if (!ok) {
        set_status(p, XS_DEV_TIMEOUT);
        *abort_flag = 1;
      }
      if (any) {  // all issued MMAs done before TMEM is released
        volatile int no_abort = 0;
        mma_commit(drain_bar);
        mbar_wait(drain_bar, 0, kWaitNs, &no_abort);
      }
    }
  } else {
    // ------------------------------------------------ epilogue (warps 2..5)
    const int q = warp & 3;                  // TMEM lane quarter of this warp
    const int row = q * 32 + lane;           // weight row inside the unit
    const bool leader = threadIdx.x == 64;
    for (int segi = 0; segi < n_seg; ++segi) {
      const Seg g = seg_at(segi);
      const long long u = g.u;
      const int k0 = g.k0, k1 = g.k1;
      const Tile tl = p.tiles[wt.tile(static_cast<int>(u / MT))];
      const int mt = static_cast<int>(u % MT);
      const int n_mma = ((tl.ntok + 15) / 16) * 16;
      const int buf = segi & 1;
      const uint32_t use = static_cast<uint32_t>(segi >> 1);
      if (leader) *s_flag = mbar_wait(accfull_bar(buf), use & 1u, kWaitNs, abort_flag) ? 1 : 0;
      named_bar_sync(1, kEpiThreads);
      const bool ok = *s_flag != 0;
      named_bar_sync(1, kEpiThreads);
      if (!ok) {
        if (leader) {
          set_status(p, XS_DEV_TIMEOUT);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const uint32_t tacc = tmem + (static_cast<uint32_t>(q * 32) << 16) + buf * C::kAccCols;
      const int col = mt * kBM + row;

      // Emits the outputs of accumulator columns [c0, c0 + 16).
      auto emit = [&](int c0, const float (&g)[16], const float (&v)[16]) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          if (c0 + j < tl.ntok) {
            const size_t r = static_cast<size_t>(tl.row0 + c0 + j) * p.M + col;
            if (kGateUp) {
              const __nv_bfloat16 h = __float2bfloat16_rn(silu(g[j]) * v[j]);
              p.act_out[r] = *reinterpret_cast<const uint16_t *>(&h);
            } else {
              p.out[r] = g[j];
            }
          }
        }
      };

      if (k0 == 0 && k1 == KI) {
        for (int c0 = 0; c0 < n_mma; c0 += 16) {
          float g[16], v[16];
          tmem_ld16(tacc + c0, g);
          if (kGateUp) tmem_ld16(tacc + 128 + c0, v);
          emit(c0, g, v);
        }
      } else {
        const int c_first = rg.cta_of(u * KI), c_last = rg.cta_of(u * KI + KI - 1);
        // Piece of a unit shared with other CTAs.  If every other piece has
        // already arrived (its sums are in its partial buffer), this one is
        // the last: it adds them to its own sums straight from TMEM, in CTA
        // order as below (same bits), without storing, fencing or arriving.
        if (leader) *s_flag = ld_acquire_gpu(p.cnt + u) == c_last - c_first ? 1 : 0;
        named_bar_sync(1, kEpiThreads);
        const bool direct_last = *s_flag != 0;
        named_bar_sync(1, kEpiThreads);
        if (direct_last) {
          __threadfence();
          for (int c0 = 0; c0 < n_mma; c0 += 16) {
            float og[16], ov[16], g[16], v[16];
            tmem_ld16(tacc + c0, og);
            if (kGateUp) tmem_ld16(tacc + 128 + c0, ov);
#pragma unroll
            for (int j = 0; j < 16; ++j) g[j] = v[j] = 0.f;
            for (int c = c_first; c <= c_last; ++c) {
              const float *src = p.part + static_cast<size_t>(c * 2 + rg.slot(c, u)) * C::kNumA * 128 * 128;
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float a = c == cta ? og[j] : __ldcg(src + (c0 + j) * 128 + row);
                g[j] = (c == c_first) ? a : g[j] + a;
                if (kGateUp) {
                  const float b = c == cta ? ov[j] : __ldcg(src + (128 + c0 + j) * 128 + row);
                  v[j] = (c == c_first) ? b : v[j] + b;
                }
              }
            }
            emit(c0, g, v);
          }
        } else {
          // Publish the partial sums.
          const int my_slot = rg.slot(cta, u);
          float *mine = p.part + static_cast<size_t>(cta * 2 + my_slot) * C::kNumA * 128 * 128;
          for (int c0 = 0; c0 < n_mma; c0 += 16) {
            float g[16], v[16];
            tmem_ld16(tacc + c0, g);
            if (kGateUp) tmem_ld16(tacc + 128 + c0, v);
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              mine[(c0 + j) * 128 + row] = g[j];
              if (kGateUp) mine[(128 + c0 + j) * 128 + row] = v[j];
            }
          }
          // The accumulator is free once the sums are in the partial buffer:
          // the MMAs of the next segment go on while this piece arrives and,
          // if it is the last, adds the pieces (from the buffers) and emits.
          __threadfence();
          tc_fence_before();
          named_bar_sync(1, kEpiThreads);
          if (leader) {
            mbar_arrive(accempty_bar(buf));
            const int old = atomicAdd(&p.cnt[u], 1);
            *s_flag = (old == c_last - c_first) ? 1 : 0;
          }
          named_bar_sync(1, kEpiThreads);
          const bool last = *s_flag != 0;
          named_bar_sync(1, kEpiThreads);
          if (last) {
            __threadfence();
            for (int c0 = 0; c0 < n_mma; c0 += 16) {
              float g[16], v[16];
#pragma unroll
              for (int j = 0; j < 16; ++j) g[j] = v[j] = 0.f;
              for (int c = c_first; c <= c_last; ++c) {
                const float *src = p.part + static_cast<size_t>(c * 2 + rg.slot(c, u)) * C::kNumA * 128 * 128;
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                  const float a = __ldcg(src + (c0 + j) * 128 + row);
                  g[j] = (c == c_first) ? a : g[j] + a;
                  if (kGateUp) {
                    const float b = __ldcg(src + (128 + c0 + j) * 128 + row);
                    v[j] = (c == c_first) ? b : v[j] + b;
                  }
                }
              }
              emit(c0, g, v);
            }
          }
          continue;  // accumulator released above
        }
      }
      tc_fence_before();
      named_bar_sync(1, kEpiThreads);
      if (leader) mbar_arrive(accempty_bar(buf));
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ---------------------------------------------------------------- host side

// Row-major [outer, inner] bf16 matrix, boxes of box_outer x 64, 128-byte swizzle.
bool make_map(CUtensorMap *m, const void *base, uint64_t inner, uint64_t outer, uint32_t box_outer) {
  return encode_tmap_2d(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, inner, outer,
                        static_cast<uint32_t>(kBK), box_outer, CU_TENSOR_MAP_SWIZZLE_128B);
}

// The token operand with boxes of 16, 32, 64 and 128 rows (one TMA per stage).
bool make_token_maps(CUtensorMap (&m)[4], const void *base, uint64_t inner, uint64_t rows) {
  for (int i = 0; i < 4; ++i)
    if (!make_map(&m[i], base, inner, rows, static_cast<uint32_t>(kBoxTok << i))) return false;
  return true;
}

template <bool kGateUp>
cudaError_t launch_phase(const TcParams &p, cudaStream_t s) {
  using C = Cfg<kGateUp>;
  cudaError_t e = cudaFuncSetAttribute(ffn_tc_kernel<kGateUp>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(ffn_tc_kernel<kGateUp>, dim3(p.grid), dim3(kThreads), C::kSmemBytes, s, p);
}

}  // namespace

size_t ffn_part_bytes(int n_sms) { return static_cast<size_t>(n_sms) * 2 * 2 * 128 * 128 * 4; }

size_t ffn_cnt_words(int max_tiles, int B, int d, int F) {
  (void)B;
  return static_cast<size_t>(max_tiles) * (F / kBM + d / kBM);
}

cudaError_t launch_ffn_gate_up(const FfnArgs &a, cudaStream_t s) {
  TcParams p;
  memset(&p, 0, sizeof(p));
  if (!make_token_maps(p.tmB, a.xp, a.d, a.max_rows)) return cudaErrorInvalidValue;
  if (a.P_gate_up != nullptr) {
    p.pk = static_cast<const uint8_t *>(a.P_gate_up);
    p.pk_shared = static_cast<const uint8_t *>(a.PS_gate_up);
  } else if (!make_map(&p.tmA0, a.W_gate, a.d, static_cast<uint64_t>(a.N) * a.F, kBM) ||
             !make_map(&p.tmA1, a.W_up, a.d, static_cast<uint64_t>(a.N) * a.F, kBM)) {
    return cudaErrorInvalidValue;
  }
  if (a.n_shared > 0 && a.P_gate_up == nullptr) {
    if (!make_map(&p.tmS0, a.S_gate, a.d, static_cast<uint64_t>(a.n_shared) * a.F, kBM) ||
        !make_map(&p.tmS1, a.S_up, a.d, static_cast<uint64_t>(a.n_shared) * a.F, kBM))
      return cudaErrorInvalidValue;
  } else if (a.P_gate_up == nullptr) {
    p.tmS0 = p.tmA0;
    p.tmS1 = p.tmA1;
  }
  p.n_routed = a.N;
  p.has_shared = a.n_shared > 0;
  p.expert_base = a.expert_base;
  p.tiles = a.tiles;
  p.meta = a.meta;
  p.stats = a.stats;
  p.part = static_cast<float *>(a.part);
  p.cnt = a.cnt;
  p.act_out = a.act;
  p.M = a.F;
  p.K = a.d;
  p.grid = a.n_sms;
  return launch_phase<true>(p, s);
}

cudaError_t launch_ffn_down(const FfnArgs &a, cudaStream_t s) {
  TcParams p;
  memset(&p, 0, sizeof(p));
  if (!make_token_maps(p.tmB, a.act, a.F, a.max_rows)) return cudaErrorInvalidValue;
  if (a.P_down != nullptr) {
    p.pk = static_cast<const uint8_t *>(a.P_down);
    p.pk_shared = static_cast<const uint8_t *>(a.PS_down);
  } else {
    if (!make_map(&p.tmA0, a.W_down, a.F, static_cast<uint64_t>(a.N) * a.d, kBM))
      return cudaErrorInvalidValue;
    p.tmA1 = p.tmA0;
    if (a.n_shared > 0) {
      if (!make_map(&p.tmS0, a.S_down, a.F, static_cast<uint64_t>(a.n_shared) * a.d, kBM))
        return cudaErrorInvalidValue;
    } else {
      p.tmS0 = p.tmA0;
    }
  }
  p.tmS1 = p.tmS0;
  p.n_routed = a.N;
  p.has_shared = a.n_shared > 0;
  p.expert_base = a.expert_base;
  p.tiles = a.tiles;
  p.meta = a.meta;
  p.stats = a.stats;
  p.part = static_cast<float *>(a.part);
  p.cnt = a.cnt + static_cast<size_t>(a.max_tiles) * (a.F / kBM);
  p.out = a.out;
  p.M = a.d;
  p.K = a.F;
  p.grid = a.n_sms;
  return launch_phase<false>(p, s);
}

}  // namespace xs
