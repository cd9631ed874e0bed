// The update that follows branch selection: group-relative advantages
// (Section 3: A_j = R_j - group mean, no standard-deviation normalisation,
// Section 4.1) and the clipped policy objective with asymmetric clipping,
// aggregated over tokens under the suffix-only masks (Sections 3.3, 4.1).
//
// Two HBM-bound launches over the packed tokens: (0) the group advantages
// and an exact integer count of the masked tokens per block (1 byte per
// token, 16-byte loads); (1) the token pass -- one warp per trajectory when
// there are many, equal token ranges per warp when there are few; either way
// the advantage is a warp-uniform scalar per trajectory and the tokens are
// streamed with 16-byte loads -- writes the final gradient (the denominator,
// folded from the counts, is known up front) and per-block fp32 sums; the
// last block to finish folds the block sums in double precision in a fixed
// order, so the loss does not depend on the timing of atomics.  The GPU's
// fp64 rate is low, so nothing per token runs in double.
#include <cuda_runtime.h>

#include <cstdint>

#include "hdl.h"
#include "hdl_internal.h"

namespace hdl {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxBlocks = 1024;

// Per-block partial sums (fp32: a block sees at most a few hundred thousand
// tokens); the grid-level fold is in double, in parallel.
struct Sums {
  float obj, tokens, clipped, ratio;
};

// Block-wide sums of four values per thread (warp shuffle trees, then
// thread 0 adds the warps' sums in order); valid in thread 0.
template <typename T>
__device__ __forceinline__ void block_sum4(T (&v)[4], T (*red)[4]) {
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) v[i] += __shfl_xor_sync(0xffffffffu, v[i], o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0)
#pragma unroll
    for (int i = 0; i < 4; ++i) red[warp][i] = v[i];
  __syncthreads();
  if (threadIdx.x == 0) {
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = red[0][i];
    for (int w = 1; w < kThreads / 32; ++w)
#pragma unroll
      for (int i = 0; i < 4; ++i) v[i] += red[w][i];
  }
}

// Bit 8i of the result is set iff byte i of w is nonzero.
__device__ __forceinline__ uint32_t nonzero_bytes(uint32_t w) {
  return (((w & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | w) >> 7 & 0x01010101u;
}

// Pass 0, one launch: the group advantages and an exact count of the
// nonzero mask bytes in [0, n), one partial count per block.
// Advantages: one warp per group, the rewards summed in double across the
// lanes, A_j = R_j - mean written per trajectory.  Count: the 16-byte-aligned
// body is read grid-stride, 16 bytes per lane and four loads per thread in
// flight; the unaligned head and tail (< 16 bytes each) by block 0, byte by
// byte.  Block 0 also resets the token pass's completion counter.
__global__ void __launch_bounds__(kThreads)
    grpo_prep_kernel(const uint8_t* __restrict__ mask, int64_t n,
                     unsigned long long* __restrict__ counts, const float* __restrict__ rewards,
                     const int32_t* __restrict__ group_offsets, int32_t n_groups, int32_t n_traj,
                     float* __restrict__ adv, unsigned int* __restrict__ done) {
  __shared__ unsigned long long red[kThreads / 32];
  if (blockIdx.x == 0 && threadIdx.x == 0) *done = 0u;
  {
    const int lane = threadIdx.x & 31;
    const int64_t nw = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
    for (int64_t g = static_cast<int64_t>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5);
         g < n_groups; g += nw) {
      int lo = group_offsets[g], hi = group_offsets[g + 1];
      lo = lo < 0 ? 0 : (lo > n_traj ? n_traj : lo);
      hi = hi < lo ? lo : (hi > n_traj ? n_traj : hi);
      if (hi == lo) continue;
      double sum = 0.0;
      for (int j = lo + lane; j < hi; j += 32) sum += rewards[j];
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      const double mean = sum / (hi - lo);
      for (int j = lo + lane; j < hi; j += 32) adv[j] = static_cast<float>(rewards[j] - mean);
    }
  }
  const int64_t head = static_cast<int64_t>((16u - (reinterpret_cast<uintptr_t>(mask) & 15u)) & 15u);
  const int64_t h = head < n ? head : n;
  const int64_t nvec = (n - h) >> 4;
  const uint4* body = reinterpret_cast<const uint4*>(mask + h);
  const int64_t tid = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x;
  const int64_t nthr = static_cast<int64_t>(gridDim.x) * kThreads;
  unsigned long long c = 0;
  int64_t v = tid;
  for (; v + 3 * nthr < nvec; v += 4 * nthr) {
    uint4 x[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) x[i] = body[v + i * nthr];
    uint32_t m = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      m += __popc(nonzero_bytes(x[i].x)) + __popc(nonzero_bytes(x[i].y)) +
           __popc(nonzero_bytes(x[i].z)) + __popc(nonzero_bytes(x[i].w));
    c += m;
  }
  for (; v < nvec; v += nthr) {
    const uint4 x = body[v];
    c += __popc(nonzero_bytes(x.x)) + __popc(nonzero_bytes(x.y)) + __popc(nonzero_bytes(x.z)) +
         __popc(nonzero_bytes(x.w));
  }
  if (blockIdx.x == 0 && n > 0) {
    const int64_t tail = h + (nvec << 4);
    if (threadIdx.x < h) c += mask[threadIdx.x] != 0;
    if (tail + threadIdx.x < n) c += mask[tail + threadIdx.x] != 0;
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long tot = 0;
    for (int w = 0; w < kThreads / 32; ++w) tot += red[w];
    counts[blockIdx.x] = tot;
  }
}

// Per-thread running sums in fp32 (a thread sees a few hundred tokens; the
// GPU's fp64 rate is far too low for a double add per token); the block fold
// is in fp32 too, the grid fold in double.
struct TokenOut {
  float obj, clipped, ratio;
};

__device__ __forceinline__ float token_grad(float lpn, float lpo, float A, float eps_low,
                                            float eps_high, float scale, TokenOut& acc) {
  const float r = expf(lpn - lpo);
  const float u = r * A;
  const float c = fminf(fmaxf(r, 1.f - eps_low), 1.f + eps_high) * A;
  const bool active = u <= c;      // the unclipped term is the minimum
  acc.obj += active ? u : c;
  acc.clipped += active ? 0.f : 1.f;
  acc.ratio += r;
  return active ? u * scale : 0.f;
}

// The trajectory holding position a: the largest j < n with offs[j] <= a
// (offsets non-decreasing, offs[0] <= a < offs[n]).  Each step the 32 lanes
// probe 32 evenly spaced candidates and keep the last one not past a, so the
// interval shrinks 32-fold per dependent load.
__device__ __forceinline__ int64_t find_traj(const int64_t* __restrict__ offs, int32_t n,
                                             int64_t a, int lane) {
  int64_t lo_j = 0, hi_j = n - 1;
  while (lo_j < hi_j) {
    const int64_t step = (hi_j - lo_j + 32) / 32;
    const int64_t c = lo_j + step * lane;
    const bool ok = c <= hi_j && offs[c] <= a;
    const unsigned m = __ballot_sync(0xffffffffu, ok);
    const int top = m ? 31 - __clz(static_cast<int>(m)) : 0;
    lo_j += step * top;
    hi_j = lo_j + step - 1 < hi_j ? lo_j + step - 1 : hi_j;
  }
  return lo_j;
}

// Token pass.  Many trajectories (kFlat = false): one warp per trajectory
// (warps loop over trajectories), its advantage a warp-uniform scalar.  Fewer
// trajectories than about twice the resident warps (kFlat = true): warp w
// takes the w-th of equal token ranges of [offs[0], offs[n]), finds the
// trajectory holding its first token and walks the trajectories it overlaps
// (their offsets and advantages read 32 at a time, one per lane), so a few
// long trajectories still keep every warp streaming.  Either way the tokens
// are streamed with 16-byte loads, three 4-token groups per lane in flight
// (64 registers: four more would cost occupancy; two measured 1 % slower).
template <bool kVec, bool kFlat>
__global__ void __launch_bounds__(kThreads, 4)
    grpo_token_kernel(const float* __restrict__ lpn, const float* __restrict__ lpo,
                      const uint8_t* __restrict__ mask, int64_t n_tokens,
                      const int64_t* __restrict__ traj_offsets, int32_t n_traj,
                      const float* __restrict__ adv, float eps_low, float eps_high,
                      const unsigned long long* __restrict__ counts, int n_count_blocks,
                      float* __restrict__ grad, Sums* __restrict__ partial,
                      unsigned int* __restrict__ done, float* __restrict__ stats, int32_t phase) {
  __shared__ float red[kThreads / 32][4];
  __shared__ double red_d[kThreads / 32][4];
  __shared__ float s_scale;
  __shared__ bool s_last;
  if (threadIdx.x < 32) {   // the denominator: an exact integer sum, one warp
    unsigned long long tot = 0;
    for (int i = threadIdx.x; i < n_count_blocks; i += 32) tot += counts[i];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    if (threadIdx.x == 0) s_scale = tot > 0 ? static_cast<float>(-1.0 / static_cast<double>(tot)) : 0.f;
  }
  __syncthreads();
  const float scale = s_scale;
  const int lane = threadIdx.x & 31;
  const int64_t lo = n_traj > 0 ? traj_offsets[0] : 0, hi = n_traj > 0 ? traj_offsets[n_traj] : 0;
  // tokens outside every trajectory carry no loss: gradient 0
  if (grad) {
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < n_tokens;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x)
      if (t < lo || t >= hi) grad[t] = 0.f;
  }
  TokenOut acc{0.f, 0.f, 0.f};
  int ntok = 0;
  // tokens [s, e) of one trajectory, advantage A: head and tail one token
  // per lane, the body three 4-token groups per lane at a time (groups start
  // at tokens p with (p + phase) % 4 == 0, where every stream is aligned)
  auto stream_trajectory = [&](int64_t s, int64_t e, float A) {
    auto one = [&](int64_t u) {
      float g = 0.f;
      if (mask[u] != 0) {
        g = token_grad(lpn[u], lpo[u], A, eps_low, eps_high, scale, acc);
        ++ntok;
      }
      if (grad) grad[u] = g;
    };
    int64_t h = s, body = s;
    if (kVec) {
      h = ((s + phase + 3) & ~int64_t{3}) - phase;
      h = h < e ? h : e;
      body = h + ((e - h) & ~int64_t{3});
    }
    if (lane < h - s) one(s + lane);
    constexpr int kBatch = kFlat ? 2 : 3;   // the flat walk holds its window too
    for (int64_t q = h; q < body; q += 4 * 32 * kBatch) {
      float4 pn[kBatch], po[kBatch];
      uint32_t mv[kBatch];
#pragma unroll
      for (int i = 0; i < kBatch; ++i) {
        const int64_t p = q + 4 * (32 * i + lane);
        mv[i] = 0u;
        if (p < body) {
          pn[i] = *reinterpret_cast<const float4*>(lpn + p);
          po[i] = *reinterpret_cast<const float4*>(lpo + p);
          mv[i] = *reinterpret_cast<const uint32_t*>(mask + p);
        }
      }
#pragma unroll
      for (int i = 0; i < kBatch; ++i) {
        const int64_t p = q + 4 * (32 * i + lane);
        if (p >= body) break;
        const float ln[4] = {pn[i].x, pn[i].y, pn[i].z, pn[i].w};
        const float l0[4] = {po[i].x, po[i].y, po[i].z, po[i].w};
        float g[4];
#pragma unroll
        for (int x = 0; x < 4; ++x) {
          g[x] = 0.f;
          if ((mv[i] >> (8 * x)) & 0xFFu) {
            g[x] = token_grad(ln[x], l0[x], A, eps_low, eps_high, scale, acc);
            ++ntok;
          }
        }
        if (grad) *reinterpret_cast<float4*>(grad + p) = make_float4(g[0], g[1], g[2], g[3]);
      }
    }
    for (int64_t u = body + lane; u < e; u += 32) one(u);
  };
  const int64_t nw = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
  const int64_t wid = static_cast<int64_t>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5);
  if constexpr (!kFlat) {
    for (int64_t j = wid; j < n_traj; j += nw) {
      int64_t ts = traj_offsets[j], te = traj_offsets[j + 1];
      ts = ts < 0 ? 0 : ts;
      te = te > n_tokens ? n_tokens : te;
      if (te > ts) stream_trajectory(ts, te, adv[j]);
    }
  } else {
    const int64_t lo_c = lo < 0 ? 0 : lo, hi_c = hi > n_tokens ? n_tokens : hi;
    const int64_t per = hi_c > lo_c ? ((hi_c - lo_c + nw - 1) / nw + 3) & ~int64_t{3} : 0;
    const int64_t a = lo_c + per * wid;
    const int64_t b = a + per < hi_c ? a + per : hi_c;
    if (a < b) {
      int64_t j = find_traj(traj_offsets, n_traj, a, lane);
      int64_t j0 = j;
      int64_t wo = traj_offsets[j0 + lane < n_traj ? j0 + lane : n_traj];
      float wa = adv[j0 + lane < n_traj ? j0 + lane : n_traj - 1];
      while (j < n_traj) {
        if (j - j0 == 31) {   // lane 31 holds only the end of the window's last trajectory
          j0 = j;
          wo = traj_offsets[j0 + lane < n_traj ? j0 + lane : n_traj];
          wa = adv[j0 + lane < n_traj ? j0 + lane : n_traj - 1];
        }
        const int i = static_cast<int>(j - j0);
        const int64_t ts = __shfl_sync(0xffffffffu, wo, i);
        const int64_t te = __shfl_sync(0xffffffffu, wo, i + 1);
        if (ts >= b) break;
        const float A = __shfl_sync(0xffffffffu, wa, i);
        const int64_t ps = ts > a ? ts : a, pe = te < b ? te : b;
        if (ps < pe) stream_trajectory(ps, pe, A);
        ++j;
      }
    }
  }
  float sf[4] = {acc.obj, static_cast<float>(ntok), acc.clipped, acc.ratio};
  block_sum4(sf, red);
  // The last block to finish folds every block's partial sums in double, in
  // a fixed order (thread i takes blocks i, i + 256, ...; then a fixed
  // tree), so the result does not depend on which block that is.
  if (threadIdx.x == 0) {
    partial[blockIdx.x] = Sums{sf[0], sf[1], sf[2], sf[3]};
    __threadfence();
    s_last = atomicAdd(done, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  double sd[4] = {0.0, 0.0, 0.0, 0.0};
  for (int b = threadIdx.x; b < static_cast<int>(gridDim.x); b += kThreads) {
    sd[0] += __ldcg(&partial[b].obj);
    sd[1] += __ldcg(&partial[b].tokens);
    sd[2] += __ldcg(&partial[b].clipped);
    sd[3] += __ldcg(&partial[b].ratio);
  }
  block_sum4(sd, red_d);
  const double o = sd[0], t = sd[1], c = sd[2], r = sd[3];
  if (threadIdx.x == 0) {
    const bool any = t > 0.0;
    stats[0] = any ? static_cast<float>(-o / t) : 0.f;
    stats[1] = static_cast<float>(t);
    stats[2] = any ? static_cast<float>(c / t) : 0.f;
    stats[3] = any ? static_cast<float>(r / t) : 0.f;
  }
}

}  // namespace
}  // namespace hdl

using namespace hdl;

extern "C" size_t hdl_grpo_loss_workspace_bytes(void) {
  return align_up(kMaxBlocks * sizeof(Sums), 256) +
         align_up(kMaxBlocks * sizeof(unsigned long long), 256) + 256;
}

extern "C" hdl_status hdl_grpo_loss(const float* logp_new, const float* logp_old,
                                    const uint8_t* mask, int64_t n_tokens,
                                    const int64_t* traj_offsets, int32_t n_traj,
                                    const float* rewards, const int32_t* group_offsets,
                                    int32_t n_groups, float eps_low, float eps_high,
                                    float* advantages, float* grad, float* stats,
                                    void* workspace, size_t workspace_bytes,
                                    void* cuda_stream) {
  HostRange range_("hdl_grpo_loss");
  if (n_tokens < 0 || n_traj < 0 || n_groups < 0) return HDL_ERR_INVALID_ARG;
  if (!(eps_low >= 0.f && eps_low < 1.f && eps_high >= 0.f)) return HDL_ERR_INVALID_ARG;
  if (!stats || (n_traj > 0 && !advantages) || (n_groups > 0 && (!rewards || !group_offsets)))
    return HDL_ERR_INVALID_ARG;
  if (n_traj > 0 && !traj_offsets) return HDL_ERR_INVALID_ARG;
  if (n_tokens > 0 && (!logp_new || !logp_old || !mask || n_traj == 0))
    return HDL_ERR_INVALID_ARG;
  if ((logp_new && !aligned_to(logp_new, 4)) || (logp_old && !aligned_to(logp_old, 4)) ||
      !aligned_to(stats, 4) || (advantages && !aligned_to(advantages, 4)) ||
      (traj_offsets && !aligned_to(traj_offsets, 8)) ||
      (group_offsets && !aligned_to(group_offsets, 4)) || (grad && !aligned_to(grad, 4)))
    return HDL_ERR_INVALID_ARG;
  if (!workspace || !aligned_to(workspace, 256) ||
      workspace_bytes < hdl_grpo_loss_workspace_bytes())
    return HDL_ERR_WORKSPACE;
  const int sms = current_sm_count();
  if (sms <= 0) return HDL_ERR_CUDA;
  cudaStream_t st = as_stream(cuda_stream);
  Sums* partial = static_cast<Sums*>(workspace);
  auto* counts = reinterpret_cast<unsigned long long*>(
      static_cast<uint8_t*>(workspace) + align_up(kMaxBlocks * sizeof(Sums), 256));
  auto* done = reinterpret_cast<unsigned int*>(
      reinterpret_cast<uint8_t*>(counts) + align_up(kMaxBlocks * sizeof(unsigned long long), 256));
  // 16-byte vectors wherever the four token streams' alignments agree
  // (buffers sliced at the same token offset included)
  const auto f_phase = [](const void* q) {
    return static_cast<int>((reinterpret_cast<uintptr_t>(q) >> 2) & 3u);
  };
  const int phase = f_phase(logp_new);
  const bool vec = n_tokens > 0 && f_phase(logp_old) == phase &&
                   static_cast<int>(reinterpret_cast<uintptr_t>(mask) & 3u) == phase &&
                   (grad == nullptr || f_phase(grad) == phase);
  // persistent grids: as many blocks as are resident at once (<= kMaxBlocks)
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, grpo_token_kernel<true, false>,
                                                    kThreads, 0) != cudaSuccess ||
      per_sm <= 0)
    per_sm = 4;
  const int64_t cap = static_cast<int64_t>(per_sm) * sms;
  // fewer trajectories than about two rounds of the resident warps: equal
  // token ranges per warp instead of one warp per trajectory
  const bool flat = n_tokens > 0 && int64_t{n_traj} < 2 * cap * (kThreads / 32);
  auto tok = vec ? (flat ? grpo_token_kernel<true, true> : grpo_token_kernel<true, false>)
                 : (flat ? grpo_token_kernel<false, true> : grpo_token_kernel<false, false>);
  // flat: at least 2048 tokens per block, up to every resident warp
  int64_t want = flat ? ceil_div(n_tokens, int64_t{2048}) : ceil_div(n_traj, kThreads / 32);
  int blocks = static_cast<int>(want < cap ? want : cap);
  if (blocks > kMaxBlocks) blocks = kMaxBlocks;
  if (blocks < 1) blocks = 1;
  // pass 0 sized by its own work: 16 KiB of mask or 8 groups per block, up
  // to 8 blocks per SM (16384 x 4096 tokens: 14.0 us against 16.7 at 4)
  want = ceil_div(n_tokens, int64_t{16384});
  const int64_t gwant = ceil_div(n_groups, kThreads / 32);
  if (gwant > want) want = gwant;
  int prep = static_cast<int>(want < 8 * sms ? want : 8 * sms);
  if (prep > kMaxBlocks) prep = kMaxBlocks;
  if (prep < 1) prep = 1;
  // the denominator counts the mask over [0, n_tokens); the token pass
  // covers the trajectories, so the two agree when the trajectories cover
  // the tokens (the documented layout)
  grpo_prep_kernel<<<prep, kThreads, 0, st>>>(mask, n_tokens, counts, rewards, group_offsets,
                                               n_groups, n_traj, advantages, done);
  if (launch_status() != HDL_OK) return HDL_ERR_CUDA;
  tok<<<blocks, kThreads, 0, st>>>(logp_new, logp_old, mask, n_tokens, traj_offsets, n_traj,
                                   advantages, eps_low, eps_high, counts, prep, grad, partial,
                                   done, stats, phase);
  return launch_status();
}
