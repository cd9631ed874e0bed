// The update that follows branch selection: group-relative advantages
// (Section 3: A_j = R_j - group mean, no standard-deviation normalisation,
// Section 4.1) and the clipped policy objective with asymmetric clipping,
// aggregated over tokens under the suffix-only masks (Sections 3.3, 4.1).
//
// Three HBM-bound passes over the packed tokens: (1) per token the ratio,
// the clipped objective and the unnormalised gradient, with per-block sums;
// (2) one block folds the block sums (double precision, fixed order, so the
// loss does not depend on atomics' timing) into the loss and statistics;
// (3) the gradient is scaled by -1 / (masked tokens).
#include <cuda_runtime.h>

#include <cstdint>

#include "hdl.h"
#include "hdl_internal.h"

namespace hdl {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxBlocks = 1024;

struct Sums {
  double obj, tokens, clipped, ratio;
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

// Last j with offs[j] <= t, in [0, n).
__device__ __forceinline__ int find_traj(const int64_t* offs, int n, int64_t t) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (offs[mid] <= t) lo = mid; else hi = mid - 1;
  }
  return lo;
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

__global__ void __launch_bounds__(kThreads)
    grpo_token_kernel(const float* __restrict__ lpn, const float* __restrict__ lpo,
                      const uint8_t* __restrict__ mask, int64_t n_tokens,
                      const int64_t* __restrict__ traj_offsets, int32_t n_traj,
                      const float* __restrict__ adv, float eps_low, float eps_high,
                      float* __restrict__ grad, Sums* __restrict__ partial) {
  __shared__ double red[kThreads / 32];
  const int64_t lo = traj_offsets[0], hi = traj_offsets[n_traj];
  double s_obj = 0.0, s_tok = 0.0, s_clip = 0.0, s_r = 0.0;
  for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < n_tokens;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float g = 0.f;
    if (mask[t] != 0 && t >= lo && t < hi) {
      const int j = find_traj(traj_offsets, n_traj, t);
      const float A = adv[j];
      const float r = expf(lpn[t] - lpo[t]);
      const float u = r * A;
      const float c = fminf(fmaxf(r, 1.f - eps_low), 1.f + eps_high) * A;
      const bool active = u <= c;      // the unclipped term is the minimum
      g = active ? u : 0.f;
      s_obj += active ? u : c;
      s_tok += 1.0;
      s_clip += active ? 0.0 : 1.0;
      s_r += r;
    }
    if (grad) grad[t] = g;
  }
  const double a = block_sum(s_obj, red);
  const double b = block_sum(s_tok, red);
  const double c = block_sum(s_clip, red);
  const double d = block_sum(s_r, red);
  if (threadIdx.x == 0) partial[blockIdx.x] = Sums{a, b, c, d};
}

__global__ void grpo_finalize_kernel(const Sums* __restrict__ partial, int n_blocks,
                                     float* __restrict__ stats, double* __restrict__ scale) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  Sums s{0.0, 0.0, 0.0, 0.0};
  for (int b = 0; b < n_blocks; ++b) {
    s.obj += partial[b].obj;
    s.tokens += partial[b].tokens;
    s.clipped += partial[b].clipped;
    s.ratio += partial[b].ratio;
  }
  const bool any = s.tokens > 0.0;
  stats[0] = any ? static_cast<float>(-s.obj / s.tokens) : 0.f;
  stats[1] = static_cast<float>(s.tokens);
  stats[2] = any ? static_cast<float>(s.clipped / s.tokens) : 0.f;
  stats[3] = any ? static_cast<float>(s.ratio / s.tokens) : 0.f;
  *scale = any ? -1.0 / s.tokens : 0.0;
}

__global__ void __launch_bounds__(kThreads)
    grpo_scale_kernel(float* __restrict__ grad, int64_t n, const double* __restrict__ scale) {
  const float k = static_cast<float>(*scale);
  for (int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; t < n;
       t += static_cast<int64_t>(gridDim.x) * blockDim.x)
    grad[t] *= k;
}

}  // namespace
}  // namespace hdl

using namespace hdl;

extern "C" size_t hdl_grpo_loss_workspace_bytes(void) {
  return align_up(kMaxBlocks * sizeof(Sums), 256) + 256;
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
  double* scale = reinterpret_cast<double*>(static_cast<uint8_t*>(workspace) +
                                            align_up(kMaxBlocks * sizeof(Sums), 256));
  if (n_groups > 0) {
    const int gb = static_cast<int>(ceil_div(n_groups, kThreads));
    group_advantage_kernel<<<gb < 4 * sms ? gb : 4 * sms, kThreads, 0, st>>>(
        rewards, group_offsets, n_groups, n_traj, advantages);
    if (launch_status() != HDL_OK) return HDL_ERR_CUDA;
  }
  int blocks = 1;
  if (n_tokens > 0) {
    const int64_t want = ceil_div(n_tokens, kThreads);
    blocks = static_cast<int>(want < kMaxBlocks ? want : kMaxBlocks);
    grpo_token_kernel<<<blocks, kThreads, 0, st>>>(logp_new, logp_old, mask, n_tokens,
                                                   traj_offsets, n_traj, advantages, eps_low,
                                                   eps_high, grad, partial);
    if (launch_status() != HDL_OK) return HDL_ERR_CUDA;
  } else {
    if (cudaMemsetAsync(partial, 0, sizeof(Sums), st) != cudaSuccess) return HDL_ERR_CUDA;
  }
  grpo_finalize_kernel<<<1, 32, 0, st>>>(partial, blocks, stats, scale);
  if (launch_status() != HDL_OK) return HDL_ERR_CUDA;
  if (grad && n_tokens > 0) {
    grpo_scale_kernel<<<blocks, kThreads, 0, st>>>(grad, n_tokens, scale);
    if (launch_status() != HDL_OK) return HDL_ERR_CUDA;
  }
  return HDL_OK;
}
