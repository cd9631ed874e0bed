// The update that follows branch selection: group-relative advantages
// (Section 3: A_j = R_j - group mean, no standard-deviation normalisation,
// Section 4.1) and the clipped policy objective with asymmetric clipping,
// aggregated over tokens under the suffix-only masks (Sections 3.3, 4.1).
//
// HBM-bound passes over the packed tokens: (0) an exact integer count of the
// masked tokens per block (1 byte per token); (1) one warp per trajectory --
// its advantage a warp-uniform scalar, its tokens streamed with 16-byte
// loads -- writes the final gradient (the denominator, folded from the
// counts, is known up front) and per-block fp32 sums; (2) one block folds
// the block sums in double precision in a fixed order, so the loss does not
// depend on the timing of atomics.  The GPU's fp64 rate is low, so nothing
// per token runs in double.
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

__global__ void group_advantage_kernel(const float* __restrict__ rewards,
                                       const int32_t* __restrict__ group_offsets,
                                       int32_t n_groups, int32_t n_traj,
                                       float* __restrict__ adv) {
  for (int g = blockIdx.x * blockDim.x + threadIdx.x; g < n_groups;
       g += gridDim.x * blockDim.x) {
    int lo = group_offsets[g], hi = group_offsets[g + 1];
    lo = lo < 0 ? 0 : (lo > n_traj ? n_traj : lo);
    hi = hi < lo ? lo : (hi > n_traj ? n_traj : hi);
    if (hi == lo) continue;
    double sum = 0.0;
    for (int j = lo; j < hi; ++j) sum += rewards[j];
    const double mean = sum / (hi - lo);
    for (int j = lo; j < hi; ++j) adv[j] = static_cast<float>(rewards[j] - mean);
  }
}

__device__ __forceinline__ float block_sum_f(float v, float* red) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float r = 0.f;
  if (threadIdx.x == 0)
    for (int w = 0; w < kThreads / 32; ++w) r += red[w];
  __syncthreads();
  return r;   // valid in thread 0
}

__device__ __forceinline__ double block_sum(double v, double* red) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  double r = 0.0;
  if (threadIdx.x == 0)
    for (int w = 0; w < kThreads / 32; ++w) r += red[w];
  __syncthreads();
  return r;   // valid in thread 0
}

// Token range of warp w of nw: contiguous, a multiple of 4 tokens long.
__device__ __forceinline__ void warp_range(int64_t lo, int64_t hi, int64_t w, int64_t nw,
                                           int64_t& a, int64_t& b) {
  const int64_t per = ((hi - lo + nw - 1) / nw + 3) & ~int64_t{3};
  a = lo + per * w;
  b = a + per < hi ? a + per : hi;
  if (a > hi) a = hi;
}

__global__ void __launch_bounds__(kThreads)
    grpo_count_kernel(const uint8_t* __restrict__ mask, int64_t lo, int64_t hi,
                      unsigned long long* __restrict__ counts) {
  __shared__ unsigned long long red[kThreads / 32];
  const int64_t nw = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
  int64_t a, b;
  warp_range(lo, hi, static_cast<int64_t>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5),
             nw, a, b);
  unsigned long long n = 0;
  for (int64_t t = a + (threadIdx.x & 31); t < b; t += 32) n += mask[t] != 0;
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = n;
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

// One warp per trajectory (warps loop over trajectories): the advantage is a
// warp-uniform scalar, the trajectory's tokens are streamed with 16-byte
// loads, two 4-token groups per lane in flight (more would cost occupancy).
template <bool kVec>
__global__ void __launch_bounds__(kThreads, 4)
    grpo_token_kernel(const float* __restrict__ lpn, const float* __restrict__ lpo,
                      const uint8_t* __restrict__ mask, int64_t n_tokens,
                      const int64_t* __restrict__ traj_offsets, int32_t n_traj,
                      const float* __restrict__ adv, float eps_low, float eps_high,
                      const unsigned long long* __restrict__ counts, int n_count_blocks,
                      float* __restrict__ grad, Sums* __restrict__ partial) {
  __shared__ float red[kThreads / 32];
  __shared__ float s_scale;
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
  const int64_t lo = traj_offsets[0], hi = traj_offsets[n_traj];
  // tokens outside every trajectory carry no loss: gradient 0
  if (grad) {
    for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < n_tokens;
         t += static_cast<int64_t>(gridDim.x) * blockDim.x)
      if (t < lo || t >= hi) grad[t] = 0.f;
  }
  TokenOut acc{0.f, 0.f, 0.f};
  int ntok = 0;
  const int64_t nw = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
  for (int64_t j = static_cast<int64_t>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5);
       j < n_traj; j += nw) {
    int64_t s = traj_offsets[j], e = traj_offsets[j + 1];
    s = s < 0 ? 0 : s;
    e = e > n_tokens ? n_tokens : e;
    if (e <= s) continue;
    const float A = adv[j];
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
      h = (s + 3) & ~int64_t{3};
      h = h < e ? h : e;
      body = h + ((e - h) & ~int64_t{3});
    }
    if (lane < h - s) one(s + lane);
    constexpr int kBatch = 2;
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
  }
  const float s0 = block_sum_f(acc.obj, red);
  const float s1 = block_sum_f(static_cast<float>(ntok), red);
  const float s2 = block_sum_f(acc.clipped, red);
  const float s3 = block_sum_f(acc.ratio, red);
  if (threadIdx.x == 0) partial[blockIdx.x] = Sums{s0, s1, s2, s3};
}

// One block folds the per-block partials in double, in a fixed order
// (thread i takes blocks i, i + 256, ...; then a fixed reduction tree).
__global__ void __launch_bounds__(kThreads)
    grpo_finalize_kernel(const Sums* __restrict__ partial, int n_blocks,
                         float* __restrict__ stats) {
  __shared__ double red[kThreads / 32];
  double o = 0.0, t = 0.0, c = 0.0, r = 0.0;
  for (int b = threadIdx.x; b < n_blocks; b += blockDim.x) {
    o += partial[b].obj;
    t += partial[b].tokens;
    c += partial[b].clipped;
    r += partial[b].ratio;
  }
  o = block_sum(o, red);
  t = block_sum(t, red);
  c = block_sum(c, red);
  r = block_sum(r, red);
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
         align_up(kMaxBlocks * sizeof(unsigned long long), 256);
}

extern "C" hdl_status hdl_grpo_loss(const float* logp_new, const float* logp_old,
                                    const uint8_t* mask, int64_t n_tokens,
                                    const int64_t* traj_offsets, int32_t n_traj,
                                    const float* rewards, const int32_t* group_offsets,
                                    int32_t n_groups, float eps_low, float eps_high,
                                    float* advantages, float* grad, float* stats,
                                    void* workspace, size_t workspace_bytes,
                                    void* cuda_stream) {
  if (n_tokens < 0 || n_traj < 0 || n_groups < 0) return HDL_ERR_INVALID_ARG;
  if (!(eps_low >= 0.f && eps_low < 1.f && eps_high >= 0.f)) return HDL_ERR_INVALID_ARG;
  if (!stats || !advantages || (n_groups > 0 && (!rewards || !group_offsets)))
    return HDL_ERR_INVALID_ARG;
  if (n_traj > 0 && !traj_offsets) return HDL_ERR_INVALID_ARG;
  if (n_tokens > 0 && (!logp_new || !logp_old || !mask || n_traj == 0))
    return HDL_ERR_INVALID_ARG;
  if (!aligned_to(stats, 4) || !aligned_to(advantages, 4) ||
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
  if (n_groups > 0) {
    const int gb = static_cast<int>(ceil_div(n_groups, kThreads));
    group_advantage_kernel<<<gb < 4 * sms ? gb : 4 * sms, kThreads, 0, st>>>(
        rewards, group_offsets, n_groups, n_traj, advantages);
    if (launch_status() != HDL_OK) return HDL_ERR_CUDA;
  }
  int blocks = 1;
  if (n_tokens > 0) {
    const bool vec = aligned_to(logp_new, 16) && aligned_to(logp_old, 16) &&
                     aligned_to(mask, 4) && (grad == nullptr || aligned_to(grad, 16));
    // persistent grids: as many blocks as are resident at once (<= kMaxBlocks)
    int per_sm = 0;
    auto tok = vec ? grpo_token_kernel<true> : grpo_token_kernel<false>;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, tok, kThreads, 0) !=
            cudaSuccess || per_sm <= 0)
      per_sm = 4;
    const int64_t cap = static_cast<int64_t>(per_sm) * sms;
    const int64_t want = ceil_div(n_traj, kThreads / 32);          // one warp per trajectory
    blocks = static_cast<int>(want < cap ? want : cap);
    if (blocks > kMaxBlocks) blocks = kMaxBlocks;
    if (blocks < 1) blocks = 1;
    // the denominator counts the mask over [0, n_tokens); the token pass
    // covers the trajectories, so the two agree when the trajectories cover
    // the tokens (the documented layout)
    grpo_count_kernel<<<blocks, kThreads, 0, st>>>(mask, 0, n_tokens, counts);
    if (launch_status() != HDL_OK) return HDL_ERR_CUDA;
    tok<<<blocks, kThreads, 0, st>>>(logp_new, logp_old, mask, n_tokens, traj_offsets, n_traj,
                                     advantages, eps_low, eps_high, counts, blocks, grad,
                                     partial);
    if (launch_status() != HDL_OK) return HDL_ERR_CUDA;
  } else {
    if (cudaMemsetAsync(partial, 0, sizeof(Sums), st) != cudaSuccess) return HDL_ERR_CUDA;
  }
  grpo_finalize_kernel<<<1, kThreads, 0, st>>>(partial, blocks, stats);
  return launch_status();
}
