// Hindsight re-scoring on the tcgen05 tensor cores (Section 3.1, Eq.
// hindsight-contexts; Section 3.2, Eq. div).
//
// For every row h of the stacked hidden states [H_orig; H_hind] (2N x d) the
// kernel needs log softmax(h W^T)[y] = z_y - log sum_v exp(z_v), z = h W^T.
// The [2N, V] logits are never stored: a persistent, warp-specialised kernel
// computes 128 x 256 logit tiles into TMEM and folds each tile straight into a
// running (max, sum of exponentials) per row, picking the target logit out of
// the tile that holds it.
//
// Work unit = (M-tile of 128 rows of one context, vocabulary chunk of up to
// 16 256-wide tiles).  Each unit writes one partial (max, sum) per row; the
// epilogue warp that publishes the last partial of a 32-token slice (every
// chunk, both contexts) merges the chunks of that slice, forming both
// log-probs, |Delta| and, when asked, the entropies -- one launch for the
// whole computation.  Units are rasterised in groups of 32 M-tiles x
// the chunks, and the chunk is sized (see geometry) so that the H and W tiles
// the ~150 concurrently running units touch stay in L2 -- W is then streamed
// from DRAM once per group instead of once per M-tile.
//
// Roles inside a CTA of 192 threads (shown for the single-CTA organisation,
// the default; Cfg below describes the CTA-pair one):
//   warp 0      TMA producer: H tile (128 x 128 B) + W tile (256 x 128 B) per
//               K step into a kStages-deep shared-memory ring;
//   warp 1      TMEM allocator and MMA issuer (one thread): 4 x
//               tcgen05.mma 128x256x(32 B) per K step, accumulators in two
//               256-column TMEM buffers so the epilogue of tile j overlaps
//               the MMAs of tile j+1;
//   warps 2..5  epilogue: one accumulator row per thread (TMEM lane), 32
//               columns per tcgen05.ld, online log-sum-exp in base 2 (and the
//               entropy numerator when asked) and the target-column select.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cfloat>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstdint>
#include <mutex>

#include "hdl.h"
#include "hdl_internal.h"
#include "ptx_sm103.cuh"

namespace hdl {
namespace {

constexpr int kBM = 128;             // rows per tile = TMEM lanes
constexpr int kBN = 256;             // vocabulary columns per tile
constexpr int kRowBytes = 128;       // K bytes per stage (one 128-byte swizzle row)
constexpr int kMaxTilesPerChunk = 16;  // up to 4096 vocabulary entries per unit
constexpr int64_t kMinUnits = 1216;     // 8 x 152: chunks shrink until this many units
constexpr double kL2Budget = 70e6;      // bytes of L2 the running units' tiles may use
constexpr int kUnitsInFlight = 152;    // work units running at once: one per SM
#ifndef HDL_GROUP_M
#define HDL_GROUP_M 32
#endif
constexpr int kGroupM = HDL_GROUP_M; // M-tiles per rasterisation group (even)
constexpr int kDefaultMode = 0;      // CTA organisation, see Cfg
constexpr int kThreads = 192;
static_assert(kGroupM % 2 == 0 && kGroupM >= 2, "group of M-tiles must be even");
constexpr int kAStage = kBM * kRowBytes;        // 16 KiB
constexpr int kMmaPerStage = kRowBytes / 32;    // 32 bytes of K per MMA
constexpr int kTmemCols = 2 * kBN;              // two accumulator buffers

// CTA organisation of the kernel:
//   mode 0  one CTA per unit, 128 x 256 MMA (cta_group::1), whole W tiles
//           (the default);
//   mode 2  clusters of two CTAs running the 256 x 256 pair MMA
//           (cta_group::2): each CTA holds its 128 H rows and one 128-row
//           half of the W tile, so a stage is 32 KiB and the ring 6 deep.
// Every copy is an ordinary tile load into the issuing CTA's own shared
// memory; no load is shared between CTAs.
template <int M>
struct Cfg {
  static_assert(M == 0 || M == 2, "CTA organisation 0 or 2");
  static constexpr bool kCluster = M == 2;
  static constexpr int kCS = M == 2 ? 2 : 1;    // CTAs per cluster
  static constexpr int kBRows = M == 2 ? kBN / 2 : kBN;  // W rows held per CTA
  static constexpr int kBStage = kBRows * kRowBytes;
  static constexpr int kStageBytes = kAStage + kBStage;
  static constexpr int kStages = M == 2 ? 6 : 4;
  static constexpr int kBarOffset = kStages * kStageBytes;
  static constexpr int kSmemBytes = kBarOffset + 256 + 1024;  // + barriers + alignment
};
constexpr uint64_t kDefaultTimeoutNs = 4000000000ull;   // 4 s per wait
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

struct RescoreArgs {
  const int32_t* targets;
  float2* part;        // [num_chunks][2N] partial (max in log2 units, sum)
  float* part_t;       // [num_chunks][2N] partial sum of p-weighted logits (entropy only)
  float* zt;           // [2N] target logit
  uint32_t* status;
  int64_t n_tokens;    // N rows per context
  int32_t vocab;
  int32_t num_kb;      // K steps (d * esize / 128)
  int32_t num_m_ctx;   // M-tiles per context
  int32_t num_m;       // M-tiles, both contexts (even)
  int32_t num_vt;      // vocabulary tiles
  int32_t num_chunks;
  int32_t tiles_per_chunk;
  int32_t num_units;   // work units (per cluster in the pair mode)
  int32_t group_m;     // M-tiles per rasterisation group (even)
  int32_t target_offset;  // targets are shifted by this (vocabulary shards)
  uint32_t inject;     // test hook: bit 0 = the producer issues no copies
  uint64_t timeout_ns;
  // Fused merge (null tile_done: the caller merges the partials itself).
  // tile_done[4 * tt + q] counts the units that have published rows
  // [128 tt + 32 q, +32) of either context; zeroed before the launch.
  uint32_t* tile_done;
  float* lp0;          // [N] log p^0
  float* lp1;          // [N] log p^H
  float* delta;        // [N] |Delta| or null
  float* ent0;         // [N] entropy of the original context or null
  float* ent1;         // [N] entropy of the hindsight context or null
};

struct Unit {
  int ctx;       // 0 = original context, 1 = hindsight context
  int row0;      // first row of the tile within its context
  int chunk;
  int vt0, vt1;  // vocabulary tiles [vt0, vt1)
};

// Grouped rasterisation: consecutive units run through group_m M-tiles
// first, then the chunks, so concurrently running units share both their
// H tiles and their W tiles in L2.  In pair mode a unit covers the two
// M-tiles 2p and 2p+1 (one per CTA of the cluster) over one chunk.
template <int kCS>
__device__ __forceinline__ Unit decode_unit(int u, const RescoreArgs& a, int rank) {
  const int tiles = (a.num_m + kCS - 1) / kCS;   // cluster tiles (last may be partly empty)
  const int gm = a.group_m / kCS > 0 ? a.group_m / kCS : 1;
  const int per_group = gm * a.num_chunks;
  const int g = u / per_group;
  const int first = g * gm;
  const int gsz = min(tiles - first, gm);
  const int r = u - g * per_group;
  const int t = first + r % gsz;
  const int mt = kCS * t + rank;   // >= num_m: an empty tile (all rows past the end)
  Unit w;
  w.chunk = r / gsz;
  w.ctx = mt >= a.num_m_ctx ? 1 : 0;
  w.row0 = (mt - w.ctx * a.num_m_ctx) * kBM;
  w.vt0 = w.chunk * a.tiles_per_chunk;
  w.vt1 = min(w.vt0 + a.tiles_per_chunk, a.num_vt);
  return w;
}

// Fold 32 logits into the running base-2 (max, sum) of one row.
__device__ __forceinline__ void lse_fold(const float (&x)[32], float& m2, float& s) {
  float c[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) c[j] = fmaxf(x[j], x[j + 16]);
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
    for (int j = 0; j < w; ++j) c[j] = fmaxf(c[j], c[j + w]);
  const float m_new = fmaxf(m2, c[0] * kLog2e);
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j & 3] += ex2_approx(fmaf(x[j], kLog2e, -m_new));
  s = fmaf(s, ex2_approx(m2 - m_new), (acc[0] + acc[1]) + (acc[2] + acc[3]));
  m2 = m_new;
}

// As lse_fold, also folding t = sum 2^(z log2e - m2) * z (the numerator of
// E_p[z], for the entropy log Z - E_p[z]).
__device__ __forceinline__ void lse_fold_ent(const float (&x)[32], float& m2, float& s,
                                             float& t) {
  float c[16];
#pragma unroll
  for (int j = 0; j < 16; ++j) c[j] = fmaxf(x[j], x[j + 16]);
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
    for (int j = 0; j < w; ++j) c[j] = fmaxf(c[j], c[j + w]);
  const float m_new = fmaxf(m2, c[0] * kLog2e);
  float acc[4] = {0.f, 0.f, 0.f, 0.f}, acct[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const float e = ex2_approx(fmaf(x[j], kLog2e, -m_new));
    acc[j & 3] += e;
    acct[j & 3] = fmaf(e, x[j], acct[j & 3]);
  }
  const float scale = ex2_approx(m2 - m_new);
  s = fmaf(s, scale, (acc[0] + acc[1]) + (acc[2] + acc[3]));
  t = fmaf(t, scale, (acct[0] + acct[1]) + (acct[2] + acct[3]));
  m2 = m_new;
}

// Merge the per-chunk partials of both contexts of token t and write
// log p^0, log p^H and |Delta| (Eq. div), and, when asked, the entropies
// H = log Z - E_p[z] of both next-token distributions.  The partials were
// written by other CTAs: they are read past L1.
template <bool kEnt>
__device__ __forceinline__ void merge_token(const RescoreArgs& a, int64_t t) {
  const int64_t n = a.n_tokens, rows_total = 2 * n;
  float lp[2], ent[2];
#pragma unroll
  for (int ctx = 0; ctx < 2; ++ctx) {
    const int64_t g = ctx * n + t;
    float M = -INFINITY;
    for (int c = 0; c < a.num_chunks; ++c) M = fmaxf(M, __ldcg(a.part + c * rows_total + g).x);
    float S = 0.f, T = 0.f;
    for (int c = 0; c < a.num_chunks; ++c) {
      const float2 p = __ldcg(a.part + c * rows_total + g);
      const float sc = exp2f(p.x - M);
      S += p.y * sc;
      if constexpr (kEnt) T += __ldcg(a.part_t + c * rows_total + g) * sc;
    }
    const float lse = (M + log2f(S)) * kLn2;
    lp[ctx] = __ldcg(a.zt + g) - lse;
    ent[ctx] = lse - T / S;
  }
  const int32_t y = __ldg(a.targets + t);
  if (y < 0 || y >= a.vocab) {
    lp[0] = lp[1] = __int_as_float(0x7fc00000);
    atomicOr(a.status, kStatusBadTarget);
  }
  a.lp0[t] = lp[0];
  a.lp1[t] = lp[1];
  if (a.delta) a.delta[t] = fabsf(lp[1] - lp[0]);
  if constexpr (kEnt) {
    if (a.ent0) a.ent0[t] = ent[0];
    if (a.ent1) a.ent1[t] = ent[1];
  }
}

// One persistent kernel for both contexts.  See Cfg for the two CTA
// organisations.  In the pair mode a stage may be refilled only once the pair
// MMAs are done with it (the even CTA commits to the stage's empty barrier in
// each CTA), both CTAs' copies are counted on the even CTA's full barrier and
// both epilogues release TMEM to the even CTA.
template <bool kTf32, int M, bool kEnt>
__global__ void __launch_bounds__(kThreads, 1)
    rescore_lse_kernel(const __grid_constant__ CUtensorMap tm_h0,
                       const __grid_constant__ CUtensorMap tm_h1,
                       const __grid_constant__ CUtensorMap tm_w, const RescoreArgs a) {
  using C = Cfg<M>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_addr(smem);
  const uint32_t sA = sbase;                          // kStages x 16 KiB
  const uint32_t sB = sbase + C::kStages * kAStage;   // kStages x kBStage
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kBarOffset);
  const uint32_t bar0 = smem_addr(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (C::kStages + s); };
  auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * C::kStages + b); };
  auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * C::kStages + 2 + b); };
  const uint32_t done_bar = bar0 + 8u * (2 * C::kStages + 4);
  uint32_t* tmem_slot =
      reinterpret_cast<uint32_t*>(smem + C::kBarOffset + 8 * (2 * C::kStages + 5));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int rank = C::kCluster ? static_cast<int>(cluster_ctarank()) : 0;
  const bool leader = rank == 0;
  const int u_first = C::kCluster ? static_cast<int>(cluster_id_x()) : static_cast<int>(blockIdx.x);
  const int u_step = C::kCluster ? static_cast<int>(cluster_count_x()) : static_cast<int>(gridDim.x);

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull_bar(b), 1);
      mbar_init(tempty_bar(b), M == 2 ? 8 : 4);
    }
    mbar_init(done_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_h0);
    tma_prefetch_desc(&tm_h1);
    tma_prefetch_desc(&tm_w);
  }
  if (warp == 1) {
    if constexpr (M == 2)
      tmem_alloc_pair(smem_addr(tmem_slot), kTmemCols);
    else
      tmem_alloc(smem_addr(tmem_slot), kTmemCols);
  }
  tc_fence_before();
  __syncthreads();
  // the peer's barriers must exist before anything is signalled into them
  if constexpr (C::kCluster) cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  PipeCtl ctl{abort_flag, a.status, a.timeout_ns};

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, pend = 0, pend_par = 0;
      bool ok = true;
      const bool stall = (a.inject & 1u) != 0;   // test hook: issue nothing
      for (int u = u_first; ok && !stall && u < a.num_units; u += u_step) {
        const Unit w = decode_unit<C::kCS>(u, a, rank);
        const CUtensorMap* tmA = w.ctx ? &tm_h1 : &tm_h0;
        for (int vt = w.vt0; ok && vt < w.vt1; ++vt) {
          for (int kb = 0; kb < a.num_kb; ++kb) {
            if (!mbar_wait_bounded(empty_bar(stage), phase ^ 1u, ctl, kRoleProducer)) {
              ok = false;
              break;
            }
            const int32_t kx = kb * (kRowBytes / (kTf32 ? 4 : 2));
            const uint32_t dA = sA + stage * kAStage, dB = sB + stage * C::kBStage;
            if constexpr (M == 2) {
              const uint32_t fb = mapa_shared(full_bar(stage), 0);
              if (leader) mbar_arrive_expect_tx(full_bar(stage), 2 * C::kStageBytes);
              tma_load_2d_pair(dA, tmA, kx, w.row0, fb);
              tma_load_2d_pair(dB, &tm_w, kx, vt * kBN + rank * (kBN / 2), fb);
            } else {
              mbar_arrive_expect_tx(full_bar(stage), C::kStageBytes);
              tma_load_2d(dA, tmA, kx, w.row0, full_bar(stage));
              tma_load_2d(dB, &tm_w, kx, vt * kBN, full_bar(stage));
            }
            pend |= 1u << stage;
            pend_par = (pend_par & ~(1u << stage)) | (phase << stage);
            if (++stage == C::kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
      if (!ok) {
        // Aborted: let the copies already issued land before the CTA exits.
        if (M == 2 && !leader) {
          // this CTA's copies are counted on the even CTA's barriers: wait a
          // bounded 2 ms, far longer than a copy takes
          const uint64_t t0 = global_timer_ns();
          while (global_timer_ns() - t0 < 2000000ull) {
          }
        } else {
          for (int s = 0; s < C::kStages; ++s)
            if ((pend >> s) & 1u)
              mbar_wait_drain(full_bar(s), (pend_par >> s) & 1u, 100000000ull);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // --------------------------------------------------------- MMA issuer
    if (lane == 0 && (M != 2 || leader)) {
      constexpr uint32_t idesc = make_idesc(kTf32 ? 2u : 1u, M == 2 ? 2 * kBM : kBM, kBN);
      int stage = 0;
      uint32_t phase = 0, tile = 0;
      bool ok = true;
      for (int u = u_first; ok && u < a.num_units; u += u_step) {
        const Unit w = decode_unit<C::kCS>(u, a, rank);
        for (int vt = w.vt0; ok && vt < w.vt1; ++vt, ++tile) {
          const uint32_t buf = tile & 1u, use = (tile >> 1) & 1u;
          if (!mbar_wait_bounded(tempty_bar(buf), use ^ 1u, ctl, kRoleMma)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + buf * kBN;
          for (int kb = 0; kb < a.num_kb; ++kb) {
            if (!mbar_wait_bounded(full_bar(stage), phase, ctl, kRoleMma)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a_addr = sA + stage * kAStage;
            const uint32_t b_addr = sB + stage * C::kBStage;
#pragma unroll
            for (int kk = 0; kk < kMmaPerStage; ++kk) {
              const uint64_t ad = smem_desc_sw128(a_addr + 32 * kk);
              const uint64_t bd = smem_desc_sw128(b_addr + 32 * kk);
              const uint32_t acc = (kb | kk) != 0 ? 1u : 0u;
              if constexpr (M == 2)
                tc_mma_pair<kTf32>(d_tmem, ad, bd, idesc, acc);
              else
                tc_mma<kTf32>(d_tmem, ad, bd, idesc, acc);
            }
            if constexpr (M == 2)
              tc_commit_pair_both(empty_bar(stage));
            else
              tc_commit(empty_bar(stage));
            if (++stage == C::kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (ok) {
            if constexpr (M == 2)
              tc_commit_pair_both(tfull_bar(buf));
            else
              tc_commit(tfull_bar(buf));
          }
        }
      }
      // Every MMA issued above (and the arrivals it feeds) must finish before
      // TMEM is released and before the peer CTA may exit.
      if constexpr (M == 2)
        tc_commit_pair(done_bar);
      else
        tc_commit(done_bar);
      mbar_wait_drain(done_bar, 0, 1000000000ull);
    }
    __syncwarp();
  } else {
    // ----------------------------------------------------------- epilogue
    const int q = warp & 3;              // TMEM lane quadrant of this warp
    const int r_in_tile = q * 32 + lane;
    const uint32_t lane_addr = static_cast<uint32_t>(q * 32) << 16;
    uint32_t tile = 0;
    bool ok = true;
    for (int u = u_first; ok && u < a.num_units; u += u_step) {
      const Unit w = decode_unit<C::kCS>(u, a, rank);
      const int64_t row = static_cast<int64_t>(w.row0) + r_in_tile;
      const bool in_range = row < a.n_tokens;
      // the target column relative to this call's vocabulary; one outside it
      // (another shard's, or a bad id) is never gathered, not even from the
      // masked tail of the last tile
      int32_t y = in_range ? __ldg(a.targets + row) - a.target_offset : -1;
      if (y < 0 || y >= a.vocab) y = -1;
      float m2 = -INFINITY, s = 0.f, zt = 0.f, tz = 0.f;
      bool found = false;
      for (int vt = w.vt0; vt < w.vt1; ++vt, ++tile) {
        const uint32_t buf = tile & 1u, use = (tile >> 1) & 1u;
        bool got = mbar_wait_bounded(tfull_bar(buf), use, ctl, kRoleEpilogue);
        if (!__all_sync(0xffffffffu, got)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int v0 = vt * kBN;
        const int ncols = min(kBN, a.vocab - v0);
        const uint32_t taddr = tmem_base + lane_addr + buf * kBN;
#pragma unroll
        for (int cc = 0; cc < kBN / 32; ++cc) {
          if (cc * 32 < ncols) {
            float x[32];
            __syncwarp();  // tcgen05.ld is warp-collective: reconverge first
            tmem_load32(taddr + cc * 32, x);
            if (cc * 32 + 32 > ncols) {
#pragma unroll
              for (int j = 0; j < 32; ++j)   // past the vocabulary: weight exactly 0
                if (cc * 32 + j >= ncols) x[j] = -FLT_MAX;
            }
            if constexpr (kEnt)
              lse_fold_ent(x, m2, s, tz);
            else
              lse_fold(x, m2, s);
            const int rel = y - (v0 + cc * 32);
            if (static_cast<unsigned>(rel) < 32u) {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (j == rel) zt = x[j];
              found = true;
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if constexpr (M == 2)
            mbar_arrive_cluster(mapa_shared(tempty_bar(buf), 0));
          else
            mbar_arrive(tempty_bar(buf));
        }
      }
      if (!ok) break;
      if (in_range) {
        const int64_t rows_total = 2 * a.n_tokens;
        const int64_t g = w.ctx * a.n_tokens + row;
        a.part[static_cast<int64_t>(w.chunk) * rows_total + g] = make_float2(m2, s);
        if constexpr (kEnt) a.part_t[static_cast<int64_t>(w.chunk) * rows_total + g] = tz;
        if (found) a.zt[g] = zt;
      }
      // Fused merge: this warp's 32 rows are published; the warp that
      // publishes the last of the 2 x num_chunks units of these rows (both
      // contexts, every chunk) merges them.  Warp-local, so a warp that gave
      // up above never leaves another one waiting.
      const int tt = w.row0 / kBM;
      if (a.tile_done != nullptr && tt < a.num_m_ctx) {
        __threadfence();
        __syncwarp();
        uint32_t prev = 0;
        if (lane == 0) prev = atomicAdd(a.tile_done + 4 * tt + q, 1u);
        prev = __shfl_sync(0xffffffffu, prev, 0);
        if (prev == 2u * static_cast<uint32_t>(a.num_chunks) - 1u) {
          // lane 0 saw every unit counted: order the lanes' reads after it
          __syncwarp();
          __threadfence();
          if (in_range) merge_token<kEnt>(a, row);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  // neither CTA of a pair may leave while the other can still write into
  // its shared memory or TMEM or arrive on its barriers
  if constexpr (C::kCluster) cluster_sync_all();
  if (warp == 1) {
    tc_fence_after();
    if constexpr (M == 2)
      tmem_dealloc_pair(tmem_base, kTmemCols);
    else
      tmem_dealloc(tmem_base, kTmemCols);
  }
}

// Per-row statistics of one vocabulary shard: the chunk partials folded to
// (m, s, zt, t): max in log2 units, sum of 2^(z log2e - m), the target logit
// (NaN when the target is outside this shard) and sum of 2^(z log2e - m) z.
__global__ void __launch_bounds__(256)
    shard_stats_kernel(const float2* __restrict__ part, const float* __restrict__ part_t,
                       const float* __restrict__ zt, int64_t n, int32_t num_chunks,
                       float4* __restrict__ stats) {
  const int64_t rows_total = 2 * n;
  for (int64_t g = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; g < rows_total;
       g += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float M = -INFINITY;
    for (int c = 0; c < num_chunks; ++c) M = fmaxf(M, part[c * rows_total + g].x);
    float S = 0.f, T = 0.f;
    for (int c = 0; c < num_chunks; ++c) {
      const float sc = exp2f(part[c * rows_total + g].x - M);
      S += part[c * rows_total + g].y * sc;
      T += part_t[c * rows_total + g] * sc;
    }
    stats[g] = make_float4(M, S, zt[g], T);
  }
}

// Merge the statistics of n_shards vocabulary shards (stats[p][ctx][t]).
__global__ void __launch_bounds__(256)
    merge_shards_kernel(const float4* __restrict__ stats, int32_t n_shards, int64_t n,
                        float* __restrict__ lp0, float* __restrict__ lp1,
                        float* __restrict__ delta, float* __restrict__ ent0,
                        float* __restrict__ ent1) {
  const int64_t rows_total = 2 * n;
  for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < n;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float lp[2], ent[2];
#pragma unroll
    for (int ctx = 0; ctx < 2; ++ctx) {
      const int64_t g = ctx * n + t;
      float M = -INFINITY;
      for (int p = 0; p < n_shards; ++p) M = fmaxf(M, stats[p * rows_total + g].x);
      float S = 0.f, T = 0.f, z = __int_as_float(0x7fc00000);
      for (int p = 0; p < n_shards; ++p) {
        const float4 q = stats[p * rows_total + g];
        const float sc = exp2f(q.x - M);
        S += q.y * sc;
        T += q.w * sc;
        if (!isnan(q.z) && isnan(z)) z = q.z;
      }
      const float lse = (M + log2f(S)) * kLn2;
      lp[ctx] = z - lse;
      ent[ctx] = lse - T / S;
    }
    lp0[t] = lp[0];
    lp1[t] = lp[1];
    if (delta) delta[t] = fabsf(lp[1] - lp[0]);
    if (ent0) ent0[t] = ent[0];
    if (ent1) ent1[t] = ent[1];
  }
}

struct Geometry {
  int64_t n;
  int esize;
  int num_kb, num_m_ctx, num_m, num_vt, num_chunks, tiles_per_chunk;
  int64_t num_units;
  size_t done_off, zt_off, part_off, part_t_off, total, total_ent;
};

// M-tiles per rasterisation group: HDL_GROUP_M (an even number in [2, 512])
// overrides kGroupM for tuning; it also sets the vocabulary chunk (see
// geometry), so results agree to rounding.
int rescore_group_m() {
  static const int g = [] {
    const char* e = std::getenv("HDL_GROUP_M");
    const int v = e ? std::atoi(e) : 0;
    return (v >= 2 && v <= 512 && v % 2 == 0) ? v : kGroupM;
  }();
  return g;
}

// HDL_CHUNK_TILES (1 ... 16) caps the vocabulary tiles per chunk, for tuning;
// results agree to rounding (the chunks' partial sums are merged in another
// grouping).
int chunk_tiles_override() {
  static const int v = [] {
    const char* e = std::getenv("HDL_CHUNK_TILES");
    const int t = e ? std::atoi(e) : 0;
    return (t >= 1 && t <= kMaxTilesPerChunk) ? t : 0;
  }();
  return v;
}

Geometry geometry(int64_t n, int32_t d, int32_t vocab, hdl_dtype dt) {
  Geometry g{};
  g.n = n;
  g.esize = dt == HDL_F32 ? 4 : 2;
  g.num_kb = static_cast<int>(static_cast<int64_t>(d) * g.esize / kRowBytes);
  g.num_m_ctx = static_cast<int>(ceil_div(n, kBM));
  g.num_m = 2 * g.num_m_ctx;
  g.num_vt = static_cast<int>(ceil_div(vocab, kBN));
  // The chunk: the largest power of two (<= 16 tiles) for which the tiles the
  // concurrently running units touch stay within kL2Budget of the 126 MB L2
  // -- the H tiles of one rasterisation group (group_m x 128 rows) plus the W
  // tiles of the chunks in flight (one chunk per group_m running units, 152
  // units running at once on 152 SMs).  Past that, W tiles
  // are evicted before the group's last units use them: on the code-shaped
  // workload 4-tile chunks (64 MB) read 90 GB from DRAM per launch instead of
  // 156 GB and run 2.5 % faster than 16-tile ones, agent-shaped (d = 5120)
  // 2-tile chunks (67 MB) 9 % faster than 4-tile ones (92 MB), and at
  // d = 4096 2-tile chunks (54 MB) up to 11 % faster than 4-tile ones
  // (73 MB): working sets from about 70 MB up were the slowest.
  const double row = static_cast<double>(d) * g.esize;
  const int gm = rescore_group_m();
  const double h_bytes = gm * static_cast<double>(kBM) * row;
  const double chunks_in_flight = static_cast<double>(kUnitsInFlight) / gm;
  g.tiles_per_chunk = kMaxTilesPerChunk;
  while (g.tiles_per_chunk > 1 &&
         h_bytes + chunks_in_flight * g.tiles_per_chunk * kBN * row > kL2Budget)
    g.tiles_per_chunk /= 2;
  // Small problems split the vocabulary finer so that every SM gets work.
  while (g.tiles_per_chunk > 1 &&
         static_cast<int64_t>(g.num_m) * ceil_div(g.num_vt, g.tiles_per_chunk) < kMinUnits)
    g.tiles_per_chunk /= 2;
  if (const int t = chunk_tiles_override(); t > 0 && t < g.tiles_per_chunk) g.tiles_per_chunk = t;
  g.num_chunks = static_cast<int>(ceil_div(g.num_vt, g.tiles_per_chunk));
  g.num_units = static_cast<int64_t>(g.num_m) * g.num_chunks;
  g.done_off = 256;   // after the status word: the fused merge's counters
  g.zt_off = g.done_off + align_up(static_cast<size_t>(g.num_m_ctx) * 4 * sizeof(uint32_t), 256);
  g.part_off = g.zt_off + align_up(static_cast<size_t>(2 * n) * sizeof(float), 256);
  g.total = g.part_off + static_cast<size_t>(g.num_chunks) * static_cast<size_t>(2 * n) * sizeof(float2);
  g.part_t_off = align_up(g.total, 256);
  g.total_ent = g.part_t_off + static_cast<size_t>(g.num_chunks) * static_cast<size_t>(2 * n) * sizeof(float);
  return g;
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// The driver's tensor-map encoder needs a context current in the calling
// thread.  A host thread whose first CUDA call is into this library has none
// yet (the library's runtime is linked statically and binds contexts lazily,
// on its first call that needs one), so bind the current device's primary
// context first -- unless the thread already has a context current.
bool ensure_context() {
  static PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
  });
  CUcontext c = nullptr;
  if (get_current && get_current(&c) == CUDA_SUCCESS && c != nullptr) return true;
  int dev = 0;
  return cudaGetDevice(&dev) == cudaSuccess && cudaSetDevice(dev) == cudaSuccess;
}

// 2-D row-major [rows, d] operand, boxes of (128 bytes of K) x box_rows,
// 128-byte swizzle; rows past the end read as zeros.
bool make_operand_map(CUtensorMap* m, const void* ptr, int64_t rows, int32_t d, int esize,
                      int box_rows) {
  auto enc = tensor_map_encoder();
  if (!enc || !ensure_context()) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(d) * esize};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kRowBytes / esize),
                       static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  // fp32 operands are loaded as TFLOAT32: the copy rounds them to tf32 to
  // nearest (measured: 4.7x smaller log-prob error than letting the tensor
  // core drop the low mantissa bits of FLOAT32 data, and no bias)
  const CUresult r = enc(m, esize == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16
                                       : CU_TENSOR_MAP_DATA_TYPE_TFLOAT32,
                         2, const_cast<void*>(ptr), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// One persistent CTA per SM (pair mode: as many clusters of two as can
// be resident at once).
template <bool kTf32, int M, bool kEnt>
hdl_status launch_rescore(const CUtensorMap& tm_h0, const CUtensorMap& tm_h1,
                          const CUtensorMap& tm_w, const RescoreArgs& a, int sms,
                          cudaStream_t st) {
  using C = Cfg<M>;
  auto kern = rescore_lse_kernel<kTf32, M, kEnt>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
      cudaSuccess)
    return HDL_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = st;
  if (C::kCluster) {
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = C::kCS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int64_t clusters = sms / C::kCS;
    cfg.gridDim = dim3(static_cast<unsigned>(C::kCS * clusters));
    int resident = 0;
    if (cudaOccupancyMaxActiveClusters(&resident, kern, &cfg) == cudaSuccess && resident > 0 &&
        resident < clusters)
      clusters = resident;
    if (clusters > a.num_units) clusters = a.num_units;
    if (clusters < 1) clusters = 1;
    cfg.gridDim = dim3(static_cast<unsigned>(C::kCS * clusters));
    if (std::getenv("HDL_PRINT_GRID"))
      std::fprintf(stderr, "hdl: mode %d grid %u (%lld clusters of %d, %d resident)\n", M,
                   cfg.gridDim.x, static_cast<long long>(clusters), C::kCS, resident);
  } else {
    cfg.gridDim = dim3(static_cast<unsigned>(a.num_units < sms ? a.num_units : sms));
  }
  if (cudaLaunchKernelEx(&cfg, kern, tm_h0, tm_h1, tm_w, a) != cudaSuccess) return HDL_ERR_CUDA;
  return HDL_OK;
}

// CTA organisation (see Cfg): kDefaultMode unless HDL_RESCORE_MODE = 0 or 2
// is set in the environment (a tuning override; both modes give the same
// results bit for bit).
int rescore_mode() {
  static const int mode = [] {
    const char* e = std::getenv("HDL_RESCORE_MODE");
    if (e && (e[0] == '0' || e[0] == '2') && e[1] == '\0') return e[0] - '0';
    return kDefaultMode;
  }();
  return mode;
}


hdl_status check_shape(int64_t n_tokens, int32_t d, int32_t vocab, hdl_dtype dt) {
  if (n_tokens < 0 || d <= 0 || vocab <= 0) return HDL_ERR_INVALID_ARG;
  if (dt != HDL_BF16 && dt != HDL_F32) return HDL_ERR_INVALID_ARG;
  if (d % 64 != 0 || d > 65536) return HDL_ERR_UNSUPPORTED;
  if (n_tokens > (int64_t{1} << 30) || vocab > (1 << 30)) return HDL_ERR_UNSUPPORTED;
  const Geometry g = geometry(n_tokens, d, vocab, dt);
  if (g.num_units >= (int64_t{1} << 31)) return HDL_ERR_UNSUPPORTED;
  return HDL_OK;
}

}  // namespace
}  // namespace hdl

using namespace hdl;

extern "C" size_t hdl_rescore_workspace_bytes(int64_t n_tokens, int32_t d, int32_t vocab,
                                              hdl_dtype dt) {
  if (check_shape(n_tokens, d, vocab, dt) != HDL_OK) return 0;
  return geometry(n_tokens, d, vocab, dt).total;
}

extern "C" size_t hdl_rescore_ex_workspace_bytes(int64_t n_tokens, int32_t d, int32_t vocab,
                                                 hdl_dtype dt, const hdl_rescore_opts* opts) {
  if (check_shape(n_tokens, d, vocab, dt) != HDL_OK) return 0;
  const Geometry g = geometry(n_tokens, d, vocab, dt);
  const bool ent = opts && (opts->entropy_orig || opts->entropy_hind);
  return ent ? g.total_ent : g.total;
}

extern "C" hdl_status hdl_rescore_ex(const void* h_orig, const void* h_hind,
                                     const void* w_lmhead, hdl_dtype dt,
                                     const int32_t* targets, int64_t n_tokens, int32_t d,
                                     int32_t vocab, float* logp_orig, float* logp_hind,
                                     float* delta, const hdl_rescore_opts* opts,
                                     void* workspace, size_t workspace_bytes,
                                     void* cuda_stream) {
  HostRange range_("hdl_rescore_ex");
  const hdl_status sh = check_shape(n_tokens, d, vocab, dt);
  if (sh != HDL_OK) return sh;
  if (n_tokens == 0) return HDL_OK;
  hdl_rescore_opts o{};
  if (opts) o = *opts;
  if (o.fault_inject & ~1u) return HDL_ERR_INVALID_ARG;
  const bool ent = o.entropy_orig || o.entropy_hind;
  if (!h_orig || !h_hind || !w_lmhead || !targets || !logp_orig || !logp_hind)
    return HDL_ERR_INVALID_ARG;
  if (!aligned_to(h_orig, 16) || !aligned_to(h_hind, 16) || !aligned_to(w_lmhead, 16) ||
      !aligned_to(targets, 4) || !aligned_to(logp_orig, 4) || !aligned_to(logp_hind, 4) ||
      (delta && !aligned_to(delta, 4)) || (o.entropy_orig && !aligned_to(o.entropy_orig, 4)) ||
      (o.entropy_hind && !aligned_to(o.entropy_hind, 4)))
    return HDL_ERR_INVALID_ARG;
  const Geometry g = geometry(n_tokens, d, vocab, dt);
  if (!workspace || !aligned_to(workspace, 256) ||
      workspace_bytes < (ent ? g.total_ent : g.total))
    return HDL_ERR_WORKSPACE;

  // the entropy variant always runs the default organisation
  const int mode = ent ? kDefaultMode : rescore_mode();
  const int cs = mode == 0 ? 1 : 2;   // CTAs per cluster
  CUtensorMap tm_h0, tm_h1, tm_w;
  if (!make_operand_map(&tm_h0, h_orig, n_tokens, d, g.esize, kBM) ||
      !make_operand_map(&tm_h1, h_hind, n_tokens, d, g.esize, kBM) ||
      !make_operand_map(&tm_w, w_lmhead, vocab, d, g.esize, kBN / cs))
    return HDL_ERR_CUDA;

  uint8_t* ws = static_cast<uint8_t*>(workspace);
  RescoreArgs a{};
  a.targets = targets;
  a.status = reinterpret_cast<uint32_t*>(ws);
  a.zt = reinterpret_cast<float*>(ws + g.zt_off);
  a.part = reinterpret_cast<float2*>(ws + g.part_off);
  a.part_t = ent ? reinterpret_cast<float*>(ws + g.part_t_off) : nullptr;
  a.n_tokens = n_tokens;
  a.vocab = vocab;
  a.num_kb = g.num_kb;
  a.num_m_ctx = g.num_m_ctx;
  a.num_m = g.num_m;
  a.num_vt = g.num_vt;
  a.num_chunks = g.num_chunks;
  a.tiles_per_chunk = g.tiles_per_chunk;
  a.num_units = static_cast<int32_t>(ceil_div(g.num_m, cs) * g.num_chunks);
  a.group_m = rescore_group_m();
  a.inject = o.fault_inject;
  a.timeout_ns = o.wait_timeout_ns ? o.wait_timeout_ns : kDefaultTimeoutNs;
  a.tile_done = reinterpret_cast<uint32_t*>(ws + g.done_off);
  a.lp0 = logp_orig;
  a.lp1 = logp_hind;
  a.delta = delta;
  a.ent0 = o.entropy_orig;
  a.ent1 = o.entropy_hind;

  cudaStream_t st = as_stream(cuda_stream);
  // the status word and the merge counters start at zero
  if (cudaMemsetAsync(ws, 0, g.zt_off, st) != cudaSuccess) return HDL_ERR_CUDA;

  const int sms = current_sm_count();
  if (sms <= 0) return HDL_ERR_CUDA;
  const bool tf32 = dt == HDL_F32;
  hdl_status ls;
  if (ent)
    ls = tf32 ? launch_rescore<true, kDefaultMode, true>(tm_h0, tm_h1, tm_w, a, sms, st)
              : launch_rescore<false, kDefaultMode, true>(tm_h0, tm_h1, tm_w, a, sms, st);
  else if (mode == 2)
    ls = tf32 ? launch_rescore<true, 2, false>(tm_h0, tm_h1, tm_w, a, sms, st)
              : launch_rescore<false, 2, false>(tm_h0, tm_h1, tm_w, a, sms, st);
  else
    ls = tf32 ? launch_rescore<true, 0, false>(tm_h0, tm_h1, tm_w, a, sms, st)
              : launch_rescore<false, 0, false>(tm_h0, tm_h1, tm_w, a, sms, st);
  if (ls != HDL_OK) return ls;
  return launch_status();
}

extern "C" hdl_status hdl_rescore(const void* h_orig, const void* h_hind, const void* w_lmhead,
                                  hdl_dtype dt, const int32_t* targets, int64_t n_tokens,
                                  int32_t d, int32_t vocab, float* logp_orig, float* logp_hind,
                                  float* delta, void* workspace, size_t workspace_bytes,
                                  void* cuda_stream) {
  return hdl_rescore_ex(h_orig, h_hind, w_lmhead, dt, targets, n_tokens, d, vocab, logp_orig,
                        logp_hind, delta, nullptr, workspace, workspace_bytes, cuda_stream);
}

extern "C" hdl_status hdl_device_status(const void* workspace, size_t workspace_bytes,
                                        void* cuda_stream, uint32_t* raw_word) {
  HostRange range_("hdl_device_status");
  if (!workspace || workspace_bytes < sizeof(uint32_t)) return HDL_ERR_INVALID_ARG;
  if (cudaStreamSynchronize(as_stream(cuda_stream)) != cudaSuccess) return HDL_ERR_CUDA;
  uint32_t word = 0;
  if (cudaMemcpy(&word, workspace, sizeof(word), cudaMemcpyDeviceToHost) != cudaSuccess)
    return HDL_ERR_CUDA;
  if (raw_word) *raw_word = word;
  if (word & kStatusTimeout) return HDL_ERR_TIMEOUT;
  if (word & kStatusBadTarget) return HDL_ERR_BAD_TARGET;
  return HDL_OK;
}

// ---------------------------------------------------------------------------
// Allocation-free variant: the scratch lives in one file-scope device array.
// Host code may not use the array's name as a device address (it is a
// host-side stand-in); its device address is looked up once per device and
// context, with that device current.
static __device__ __align__(256) uint8_t g_static_scratch[HDL_STATIC_SCRATCH_BYTES];

namespace {
constexpr int kMaxDevices = 128;
std::mutex g_scratch_mu;
struct ScratchSlot {
  unsigned long long ctx_id;   // the context the address belongs to (0 = none yet)
  void* addr;
};
ScratchSlot g_scratch[kMaxDevices] = {};

// Process-unique id of the calling thread's current context (never reused,
// unlike a context handle, so a context re-created after cudaDeviceReset has
// a new one); 0 if it cannot be read.
unsigned long long current_context_id() {
  static PFN_cuCtxGetId_v12000 get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(p);
  });
  unsigned long long id = 0;
  if (!get_id || get_id(nullptr, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// The array's device address in the current device's current context.  The
// address is cached per device together with the context's id; a call from
// another context of the device (e.g. after cudaDeviceReset re-created the
// primary context) looks it up again.
hdl_status static_scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return HDL_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return HDL_ERR_UNSUPPORTED;
  if (!ensure_context()) return HDL_ERR_CUDA;
  const unsigned long long ctx = current_context_id();
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  ScratchSlot& slot = g_scratch[dev];
  if (ctx == 0 || slot.addr == nullptr || slot.ctx_id != ctx) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr)
      return HDL_ERR_CUDA;
    slot.addr = p;
    slot.ctx_id = ctx;
  }
  *out = slot.addr;
  return HDL_OK;
}
}  // namespace

extern "C" hdl_status hdl_rescore_noalloc(const void* h_orig, const void* h_hind,
                                          const void* w_lmhead, hdl_dtype dt,
                                          const int32_t* targets, int64_t n_tokens, int32_t d,
                                          int32_t vocab, float* logp_orig, float* logp_hind,
                                          float* delta, const void** scratch_out,
                                          void* cuda_stream) {
  HostRange range_("hdl_rescore_noalloc");
  const hdl_status sh = check_shape(n_tokens, d, vocab, dt);
  if (sh != HDL_OK) return sh;
  if (n_tokens == 0) return HDL_OK;
  if (geometry(n_tokens, d, vocab, dt).total > HDL_STATIC_SCRATCH_BYTES)
    return HDL_ERR_UNSUPPORTED;
  void* ws = nullptr;
  const hdl_status st = static_scratch_address(&ws);
  if (st != HDL_OK) return st;
  if (scratch_out) *scratch_out = ws;
  return hdl_rescore(h_orig, h_hind, w_lmhead, dt, targets, n_tokens, d, vocab, logp_orig,
                     logp_hind, delta, ws, HDL_STATIC_SCRATCH_BYTES, cuda_stream);
}

// ---------------------------------------------------------------------------
// Vocabulary-parallel re-scoring: one shard of W per call, statistics out.
extern "C" size_t hdl_rescore_shard_workspace_bytes(int64_t n_tokens, int32_t d,
                                                    int32_t vocab_shard, hdl_dtype dt) {
  if (check_shape(n_tokens, d, vocab_shard, dt) != HDL_OK) return 0;
  return geometry(n_tokens, d, vocab_shard, dt).total_ent;
}

extern "C" hdl_status hdl_rescore_shard(const void* h_orig, const void* h_hind,
                                        const void* w_shard, hdl_dtype dt,
                                        const int32_t* targets, int64_t n_tokens, int32_t d,
                                        int32_t vocab_shard, int32_t vocab_offset, float* stats,
                                        void* workspace, size_t workspace_bytes,
                                        void* cuda_stream) {
  HostRange range_("hdl_rescore_shard");
  const hdl_status sh = check_shape(n_tokens, d, vocab_shard, dt);
  if (sh != HDL_OK) return sh;
  if (vocab_offset < 0) return HDL_ERR_INVALID_ARG;
  if (n_tokens == 0) return HDL_OK;
  if (!h_orig || !h_hind || !w_shard || !targets || !stats) return HDL_ERR_INVALID_ARG;
  if (!aligned_to(h_orig, 16) || !aligned_to(h_hind, 16) || !aligned_to(w_shard, 16) ||
      !aligned_to(targets, 4) || !aligned_to(stats, 16))
    return HDL_ERR_INVALID_ARG;
  const Geometry g = geometry(n_tokens, d, vocab_shard, dt);
  if (!workspace || !aligned_to(workspace, 256) || workspace_bytes < g.total_ent)
    return HDL_ERR_WORKSPACE;
  constexpr int cs = Cfg<kDefaultMode>::kCS;
  CUtensorMap tm_h0, tm_h1, tm_w;
  if (!make_operand_map(&tm_h0, h_orig, n_tokens, d, g.esize, kBM) ||
      !make_operand_map(&tm_h1, h_hind, n_tokens, d, g.esize, kBM) ||
      !make_operand_map(&tm_w, w_shard, vocab_shard, d, g.esize, kBN / cs))
    return HDL_ERR_CUDA;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  RescoreArgs a{};
  a.targets = targets;
  a.status = reinterpret_cast<uint32_t*>(ws);
  a.zt = reinterpret_cast<float*>(ws + g.zt_off);
  a.part = reinterpret_cast<float2*>(ws + g.part_off);
  a.part_t = reinterpret_cast<float*>(ws + g.part_t_off);
  a.n_tokens = n_tokens;
  a.vocab = vocab_shard;
  a.num_kb = g.num_kb;
  a.num_m_ctx = g.num_m_ctx;
  a.num_m = g.num_m;
  a.num_vt = g.num_vt;
  a.num_chunks = g.num_chunks;
  a.tiles_per_chunk = g.tiles_per_chunk;
  a.num_units = static_cast<int32_t>(ceil_div(g.num_m, cs) * g.num_chunks);
  a.group_m = rescore_group_m();
  a.target_offset = vocab_offset;
  a.timeout_ns = kDefaultTimeoutNs;
  cudaStream_t st = as_stream(cuda_stream);
  if (cudaMemsetAsync(a.status, 0, sizeof(uint32_t), st) != cudaSuccess) return HDL_ERR_CUDA;
  // rows whose target this shard does not hold keep a NaN target logit
  if (cudaMemsetAsync(a.zt, 0xFF, static_cast<size_t>(2 * n_tokens) * sizeof(float), st) !=
      cudaSuccess)
    return HDL_ERR_CUDA;
  const int sms = current_sm_count();
  if (sms <= 0) return HDL_ERR_CUDA;
  const hdl_status ls =
      dt == HDL_F32 ? launch_rescore<true, kDefaultMode, true>(tm_h0, tm_h1, tm_w, a, sms, st)
                    : launch_rescore<false, kDefaultMode, true>(tm_h0, tm_h1, tm_w, a, sms, st);
  if (ls != HDL_OK) return ls;
  if (launch_status() != HDL_OK) return HDL_ERR_CUDA;
  const int64_t blocks = ceil_div(2 * n_tokens, 256);
  const int grid = static_cast<int>(blocks < 8 * sms ? blocks : 8 * sms);
  shard_stats_kernel<<<grid, 256, 0, st>>>(a.part, a.part_t, a.zt, n_tokens, g.num_chunks,
                                           reinterpret_cast<float4*>(stats));
  return launch_status();
}

extern "C" hdl_status hdl_merge_vocab_shards(const float* stats, int32_t n_shards,
                                             int64_t n_tokens, float* logp_orig,
                                             float* logp_hind, float* delta,
                                             float* entropy_orig, float* entropy_hind,
                                             void* cuda_stream) {
  HostRange range_("hdl_merge_vocab_shards");
  if (n_shards <= 0 || n_tokens < 0) return HDL_ERR_INVALID_ARG;
  if (n_tokens == 0) return HDL_OK;
  if (!stats || !logp_orig || !logp_hind) return HDL_ERR_INVALID_ARG;
  if (!aligned_to(stats, 16) || !aligned_to(logp_orig, 4) || !aligned_to(logp_hind, 4) ||
      (delta && !aligned_to(delta, 4)) || (entropy_orig && !aligned_to(entropy_orig, 4)) ||
      (entropy_hind && !aligned_to(entropy_hind, 4)))
    return HDL_ERR_INVALID_ARG;
  const int sms = current_sm_count();
  if (sms <= 0) return HDL_ERR_CUDA;
  const int64_t blocks = ceil_div(n_tokens, 256);
  const int grid = static_cast<int>(blocks < 8 * sms ? blocks : 8 * sms);
  merge_shards_kernel<<<grid, 256, 0, as_stream(cuda_stream)>>>(
      reinterpret_cast<const float4*>(stats), n_shards, n_tokens, logp_orig, logp_hind, delta,
      entropy_orig, entropy_hind);
  return launch_status();
}
