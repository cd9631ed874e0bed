// Branch-point selection (Section 3.2: rank each root's candidate positions by
// the hindsight-divergence score and take the highest; Section 3.1: only
// policy-generated tokens are candidates; Section 4.4: of points too close
// together only one is kept).
//
// One CTA per root.  A candidate is encoded as a 64-bit key whose order is
// the ranking: high word = the score mapped to an order-preserving unsigned
// integer (-0 folded onto +0), low word = ~t, so that equal scores rank the
// lower position first.  Key 0 never occurs for a real candidate and means
// "none".
//   plain top-k: each thread keeps a sorted register list of its 16 best
//     keys while streaming its strided share of the root; then k rounds of a
//     block-wide max pick the winners, the owning thread popping its head.
//   greedy spacing (gap_mode 0): k rounds, each a full scan for the best key
//     not within min_gap of an accepted point (the greedy walk of the ranked
//     list accepts exactly these points in this order).
//   drop-lower spacing (gap_mode 1): plain top-k, then thread 0 walks the k
//     points in rank order and keeps those not too close to a kept one.
#include <cuda_runtime.h>

#include <cstdint>

#include "hdl.h"
#include "hdl_internal.h"

namespace hdl {
namespace {

constexpr int kSelThreads = 512;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kMaxK = 16;

__device__ __forceinline__ uint32_t score_order(float f) {
  uint32_t u = __float_as_uint(f);
  if (u == 0x80000000u) u = 0u;  // -0 ranks like +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ uint64_t make_key(float score, int64_t t) {
  return (static_cast<uint64_t>(score_order(score)) << 32) |
         static_cast<uint64_t>(0xFFFFFFFFu - static_cast<uint32_t>(t));
}

__device__ __forceinline__ int64_t key_pos(uint64_t key) {
  return static_cast<int64_t>(0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFu));
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    const uint64_t w = __shfl_xor_sync(0xffffffffu, v, o);
    v = w > v ? w : v;
  }
  return v;
}

// Block-wide max of one key per thread; every thread gets the result.
__device__ __forceinline__ uint64_t block_max_u64(uint64_t v, uint64_t* red) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  v = warp_max_u64(v);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  if (warp == 0) {
    uint64_t x = lane < kSelWarps ? red[lane] : 0ull;
    x = warp_max_u64(x);
    if (lane == 0) red[kSelWarps] = x;
  }
  __syncthreads();
  const uint64_t r = red[kSelWarps];
  __syncthreads();  // red[] is reused by the next call
  return r;
}

struct RootView {
  int64_t start;   // absolute index of the root's first token
  int64_t w_lo, w_hi;  // candidate window, root-relative
};

__device__ __forceinline__ bool is_candidate(const float* delta, const uint8_t* valid,
                                             int64_t n_tokens, int64_t abs_t, float& s) {
  if (abs_t < 0 || abs_t >= n_tokens) return false;
  if (valid && valid[abs_t] == 0) return false;
  s = delta[abs_t];
  return !isnan(s);
}

__global__ void __launch_bounds__(kSelThreads)
    select_branches_kernel(const float* __restrict__ delta, const uint8_t* __restrict__ valid,
                           int64_t n_tokens, const int64_t* __restrict__ root_offsets,
                           int32_t n_roots, int32_t k, int32_t min_gap, int32_t gap_mode,
                           int32_t lo, int32_t hi, int32_t* __restrict__ branch_pos,
                           int32_t* __restrict__ n_selected, float* __restrict__ branch_delta) {
  __shared__ uint64_t red[kSelWarps + 1];
  __shared__ int64_t chosen[kMaxK];
  __shared__ int n_chosen;

  for (int r = blockIdx.x; r < n_roots; r += gridDim.x) {
    const int64_t start = root_offsets[r];
    const int64_t end = root_offsets[r + 1];
    const int64_t T = end > start ? end - start : 0;
    const int64_t w_lo = lo > 0 ? lo : 0;
    const int64_t w_hi = hi <= 0 ? T : (hi < T ? hi : T);
    if (threadIdx.x == 0) n_chosen = 0;
    __syncthreads();

    if (min_gap <= 0 || gap_mode == 1) {
      // plain top-k (also the first stage of drop-lower)
      uint64_t top[kMaxK];
#pragma unroll
      for (int j = 0; j < kMaxK; ++j) top[j] = 0ull;
      for (int64_t t = w_lo + threadIdx.x; t < w_hi; t += kSelThreads) {
        float s;
        if (!is_candidate(delta, valid, n_tokens, start + t, s)) continue;
        const uint64_t key = make_key(s, t);
        if (key > top[kMaxK - 1]) {
#pragma unroll
          for (int j = kMaxK - 1; j > 0; --j)
            top[j] = key > top[j - 1] ? top[j - 1] : (key > top[j] ? key : top[j]);
          top[0] = key > top[0] ? key : top[0];
        }
      }
      for (int j = 0; j < k; ++j) {
        const uint64_t best = block_max_u64(top[0], red);
        if (best == 0ull) break;
        if (top[0] == best) {
#pragma unroll
          for (int i = 0; i < kMaxK - 1; ++i) top[i] = top[i + 1];
          top[kMaxK - 1] = 0ull;
        }
        if (threadIdx.x == 0) chosen[n_chosen++] = key_pos(best);
      }
      __syncthreads();
      if (min_gap > 0 && threadIdx.x == 0) {
        // drop-lower: keep, in rank order, the points not too close to a kept one
        int kept = 0;
        for (int i = 0; i < n_chosen; ++i) {
          bool close = false;
          for (int j = 0; j < kept; ++j) {
            const int64_t dd = chosen[i] - chosen[j];
            if ((dd < 0 ? -dd : dd) < min_gap) close = true;
          }
          if (!close) chosen[kept++] = chosen[i];
        }
        n_chosen = kept;
      }
    } else {
      // greedy spacing: each round takes the best point compatible with all
      // points accepted so far
      for (int j = 0; j < k; ++j) {
        const int na = n_chosen;
        uint64_t mine = 0ull;
        for (int64_t t = w_lo + threadIdx.x; t < w_hi; t += kSelThreads) {
          float s;
          if (!is_candidate(delta, valid, n_tokens, start + t, s)) continue;
          bool close = false;
          for (int i = 0; i < na; ++i) {
            const int64_t dd = t - chosen[i];
            if ((dd < 0 ? -dd : dd) < min_gap) close = true;
          }
          if (close) continue;
          const uint64_t key = make_key(s, t);
          mine = key > mine ? key : mine;
        }
        const uint64_t best = block_max_u64(mine, red);
        if (best == 0ull) break;
        if (threadIdx.x == 0) {
          chosen[n_chosen] = key_pos(best);
          n_chosen = n_chosen + 1;
        }
        __syncthreads();
      }
    }
    __syncthreads();
    if (threadIdx.x < k) {
      const int j = threadIdx.x;
      const int n = n_chosen;
      const int64_t o = static_cast<int64_t>(r) * k + j;
      if (j < n) {
        branch_pos[o] = static_cast<int32_t>(chosen[j]);
        if (branch_delta) branch_delta[o] = delta[start + chosen[j]];
      } else {
        branch_pos[o] = -1;
        if (branch_delta) branch_delta[o] = __int_as_float(0x7fc00000);
      }
      if (j == 0) n_selected[r] = n;
    }
    if (k == 0 && threadIdx.x == 0) n_selected[r] = 0;
    __syncthreads();
  }
}

}  // namespace
}  // namespace hdl

using namespace hdl;

extern "C" hdl_status hdl_select_branches(const float* delta, const uint8_t* valid,
                                          int64_t n_tokens, const int64_t* root_offsets,
                                          int32_t n_roots, int32_t k,
                                          const hdl_select_opts* opts, int32_t* branch_pos,
                                          int32_t* n_selected, float* branch_delta,
                                          void* cuda_stream) {
  if (n_roots < 0 || n_tokens < 0 || k < 0) return HDL_ERR_INVALID_ARG;
  if (k > kMaxK) return HDL_ERR_UNSUPPORTED;
  hdl_select_opts o{0, 0, 0, 0};
  if (opts) o = *opts;
  if (o.min_gap < 0 || (o.gap_mode != 0 && o.gap_mode != 1)) return HDL_ERR_INVALID_ARG;
  if (n_roots == 0) return HDL_OK;
  if (!root_offsets || !n_selected || (k > 0 && !branch_pos) || (n_tokens > 0 && !delta))
    return HDL_ERR_INVALID_ARG;
  if (!aligned_to(root_offsets, 8) || !aligned_to(n_selected, 4) ||
      (branch_pos && !aligned_to(branch_pos, 4)) || (delta && !aligned_to(delta, 4)) ||
      (branch_delta && !aligned_to(branch_delta, 4)))
    return HDL_ERR_INVALID_ARG;
  const int sms = current_sm_count();
  if (sms <= 0) return HDL_ERR_CUDA;
  const int grid = n_roots < 32 * sms ? n_roots : 32 * sms;
  select_branches_kernel<<<grid, kSelThreads, 0, as_stream(cuda_stream)>>>(
      delta, valid, n_tokens, root_offsets, n_roots, k, o.min_gap, o.gap_mode, o.lo, o.hi,
      branch_pos, n_selected, branch_delta);
  return launch_status();
}
