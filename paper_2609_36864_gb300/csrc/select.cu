// Branch-point selection (Section 3.2: rank each root's candidate positions by
// the hindsight-divergence score and take the highest; Section 3.1: only
// policy-generated tokens are candidates; Section 4.4: of points too close
// together only one is kept).
//
// A candidate is encoded as a 64-bit key whose order is the ranking: high
// word = the score mapped to an order-preserving unsigned integer (-0 folded
// onto +0), low word = ~t, so that equal scores rank the lower position
// first.  Key 0 never occurs for a real candidate and means "none".
//
// Plain top-k (the default): select_topk_kernel streams each root with
// 16-byte loads (4 scores + 4 validity bytes per lane) into one exact top-k
// list per warp held across its lanes; a candidate is compared with the
// current k-th best and only the few that beat it (about k ln(T/k) per root)
// are inserted, cooperatively (ballot + shuffle), so no lane ever runs a
// divergent insertion.  One warp per root when there are many roots, one
// block of 16 warps per root (the per-warp lists merged by warp 0) when there
// are few long ones.
// Spacing rule (min_gap > 0): select_spacing_kernel, one CTA per root --
//   greedy (gap_mode 0): k rounds, each a full scan for the best key not
//     within min_gap of an accepted point (the greedy walk of the ranked
//     list accepts exactly these points in this order);
//   drop-lower (gap_mode 1): plain top-k, then thread 0 walks the k points
//     in rank order and keeps those not too close to a kept one.
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

__device__ __forceinline__ bool is_candidate(const float* delta, const uint8_t* valid,
                                             int64_t n_tokens, int64_t abs_t, float& s) {
  if (abs_t < 0 || abs_t >= n_tokens) return false;
  if (valid && valid[abs_t] == 0) return false;
  s = delta[abs_t];
  return !isnan(s);
}

__global__ void __launch_bounds__(kSelThreads)
    select_spacing_kernel(const float* __restrict__ delta, const uint8_t* __restrict__ valid,
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

// The warp's running top-k is distributed over its lanes: lane j < k holds
// the j-th best key so far (0 = empty), lanes >= k hold 0.  tau = lane k-1's
// key is the exact k-th best; a candidate must beat it to enter.
struct WarpTopK {
  uint64_t mine;   // this lane's entry
  uint64_t tau;    // k-th best so far, on every lane
  float tau_s;     // its score (-inf while the list is not full)
};

// Inverse of score_order on a key's high word.
__device__ __forceinline__ float key_score(uint64_t key) {
  if (key == 0ull) return -INFINITY;
  const uint32_t u = static_cast<uint32_t>(key >> 32);
  return __uint_as_float((u & 0x80000000u) ? (u ^ 0x80000000u) : ~u);
}

// Insert `key` (> tau, identical on every lane) into the list.
__device__ __forceinline__ void wtk_insert(WarpTopK& w, uint64_t key, int k, int lane) {
  const int pos = __popc(__ballot_sync(0xffffffffu, w.mine > key));
  const uint64_t prev = __shfl_up_sync(0xffffffffu, w.mine, 1);
  if (lane > pos) w.mine = prev;
  if (lane == pos) w.mine = key;
  if (lane >= k) w.mine = 0ull;
  w.tau = __shfl_sync(0xffffffffu, w.mine, k - 1);
  w.tau_s = key_score(w.tau);
}

// Offer each lane's candidate (score s at root position t; ok = valid): a
// candidate whose score is below the k-th best's is rejected by one float
// compare (it cannot beat tau); the few others get their key built (NaN
// scores get none) and are inserted one at a time, lowest lane first, each
// re-tested against the new tau.
__device__ __forceinline__ void wtk_offer_key(WarpTopK& w, uint64_t key, int k, int lane) {
  unsigned pending = __ballot_sync(0xffffffffu, key > w.tau);
  while (pending) {
    const int src = __ffs(pending) - 1;
    const uint64_t cand = __shfl_sync(0xffffffffu, key, src);
    wtk_insert(w, cand, k, lane);
    if (lane == src) key = 0ull;
    pending = __ballot_sync(0xffffffffu, key > w.tau);
  }
}

__device__ __forceinline__ void wtk_offer(WarpTopK& w, float s, bool ok, int64_t t, int k,
                                          int lane) {
  ok = ok && s >= w.tau_s;
  if (!__any_sync(0xffffffffu, ok)) return;
  wtk_offer_key(w, ok && !isnan(s) ? make_key(s, t) : 0ull, k, lane);
}

// The warp streams absolute positions [a0, a1) of the root starting at
// `start`: scalar head and tail, and a vector body walked in warp-uniform
// steps of 4 x 32 four-position groups whose loads are all issued first.
template <bool kVec>
__device__ __forceinline__ void stream_range(WarpTopK& w, const float* delta, const uint8_t* valid,
                                             int64_t start, int64_t a0, int64_t a1, int k,
                                             int lane) {
  if (!kVec) {
    for (int64_t q = a0; q < a1; q += 32) {
      const int64_t p = q + lane;
      const bool in = p < a1;
      wtk_offer(w, in ? delta[p] : 0.f, in && (valid == nullptr || valid[p] != 0), p - start, k,
                lane);
    }
    return;
  }
  const int64_t h = a0 + ((4 - (a0 & 3)) & 3) < a1 ? a0 + ((4 - (a0 & 3)) & 3) : a1;
  {
    const int64_t p = a0 + lane;
    const bool in = p < h;
    wtk_offer(w, in ? delta[p] : 0.f, in && (valid == nullptr || valid[p] != 0), p - start, k,
              lane);
  }
  const int64_t body = h + ((a1 - h) & ~int64_t{3});
  constexpr int kBatch = 4;
  for (int64_t q = h; q < body; q += 4 * 32 * kBatch) {
    float4 d[kBatch];
    uint32_t v[kBatch];
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
      const int64_t p = q + 4 * (32 * i + lane);
      if (p < body) {
        d[i] = *reinterpret_cast<const float4*>(delta + p);
        v[i] = valid ? *reinterpret_cast<const uint32_t*>(valid + p) : 0x01010101u;
      } else {
        d[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        v[i] = 0u;
      }
    }
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
      const int64_t t = q + 4 * (32 * i + lane) - start;
      wtk_offer(w, d[i].x, (v[i] & 0xFFu) != 0, t, k, lane);
      wtk_offer(w, d[i].y, (v[i] & 0xFF00u) != 0, t + 1, k, lane);
      wtk_offer(w, d[i].z, (v[i] & 0xFF0000u) != 0, t + 2, k, lane);
      wtk_offer(w, d[i].w, (v[i] & 0xFF000000u) != 0, t + 3, k, lane);
    }
  }
  {
    const int64_t p = body + lane;
    const bool in = p < a1;
    wtk_offer(w, in ? delta[p] : 0.f, in && (valid == nullptr || valid[p] != 0), p - start, k,
              lane);
  }
}

// kWarps == 1: one warp per root (8 roots per 256-thread block);
// kWarps == 16: one block per root, each warp a contiguous slice, the
// partial lists merged by warp 0 through shared memory.
template <int kWarps, bool kVec>
__global__ void __launch_bounds__(kWarps == 1 ? 256 : 32 * kWarps)
    select_topk_kernel(const float* __restrict__ delta, const uint8_t* __restrict__ valid,
                       int64_t n_tokens, const int64_t* __restrict__ root_offsets,
                       int32_t n_roots, int32_t k, int32_t lo, int32_t hi,
                       int32_t* __restrict__ branch_pos, int32_t* __restrict__ n_selected,
                       float* __restrict__ branch_delta) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int roots_per_block = kWarps == 1 ? blockDim.x / 32 : 1;
  const int64_t first =
      static_cast<int64_t>(blockIdx.x) * roots_per_block + (kWarps == 1 ? warp : 0);
  const int64_t step = static_cast<int64_t>(gridDim.x) * roots_per_block;
  __shared__ uint64_t lists[kWarps == 1 ? 1 : kWarps][32];
  for (int64_t r = first; r < n_roots; r += step) {
    const int64_t start = root_offsets[r];
    const int64_t end = root_offsets[r + 1];
    const int64_t T = end > start ? end - start : 0;
    const int64_t w_lo = lo > 0 ? lo : 0;
    const int64_t w_hi = hi <= 0 ? T : (hi < T ? hi : T);
    int64_t a0 = start + w_lo, a1 = start + w_hi;
    if (a0 < 0) a0 = 0;
    if (a1 > n_tokens) a1 = n_tokens;
    WarpTopK w{0ull, 0ull, -INFINITY};
    if (kWarps == 1) {
      if (a1 > a0) stream_range<kVec>(w, delta, valid, start, a0, a1, k, lane);
    } else {
      const int64_t len = a1 > a0 ? a1 - a0 : 0;
      const int64_t per = ((len + kWarps - 1) / kWarps + 3) & ~int64_t{3};
      const int64_t s0 = a0 + per * warp;
      const int64_t s1 = s0 + per < a1 ? s0 + per : a1;
      if (s0 < s1) stream_range<kVec>(w, delta, valid, start, s0, s1, k, lane);
      lists[warp][lane] = w.mine;
      __syncthreads();
      if (warp == 0) {
        w = WarpTopK{0ull, 0ull, -INFINITY};
        for (int i = 0; i < kWarps; ++i) wtk_offer_key(w, lists[i][lane], k, lane);
      }
      __syncthreads();
      if (warp != 0) continue;
    }
    const int n = __popc(__ballot_sync(0xffffffffu, w.mine != 0ull));
    if (lane < k) {
      const int64_t o = r * k + lane;
      if (lane < n) {
        const int64_t t = key_pos(w.mine);
        branch_pos[o] = static_cast<int32_t>(t);
        if (branch_delta) branch_delta[o] = delta[start + t];
      } else {
        branch_pos[o] = -1;
        if (branch_delta) branch_delta[o] = __int_as_float(0x7fc00000);
      }
    }
    if (lane == 0) n_selected[r] = n;
  }
}

// Many roots: one warp per root, a persistent grid of as many 8-warp blocks
// as are resident at once.  Few roots: 16 warps per root so that the GPU
// fills.  (Splitting mid-length roots over 4 warps was measured slower: the
// per-root barrier and merge cost more than the shorter chains save.)
template <bool kVec>
hdl_status launch_topk(const float* delta, const uint8_t* valid, int64_t n_tokens,
                       const int64_t* offs, int32_t n_roots, int32_t k, int32_t lo, int32_t hi,
                       int32_t* bp, int32_t* ns, float* bd, int sms, cudaStream_t st) {
  if (n_roots >= 2 * sms) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, select_topk_kernel<1, kVec>, 256,
                                                      0) != cudaSuccess || per_sm <= 0)
      per_sm = 4;
    const int64_t blocks = (n_roots + 7) / 8;
    const int64_t cap = static_cast<int64_t>(per_sm) * sms;
    const int grid = static_cast<int>(blocks < cap ? blocks : cap);
    select_topk_kernel<1, kVec><<<grid, 256, 0, st>>>(delta, valid, n_tokens, offs, n_roots, k,
                                                      lo, hi, bp, ns, bd);
  } else {
    select_topk_kernel<16, kVec><<<n_roots, 512, 0, st>>>(delta, valid, n_tokens, offs,
                                                          n_roots, k, lo, hi, bp, ns, bd);
  }
  return launch_status();
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
  if (n_tokens >= (int64_t{1} << 31)) return HDL_ERR_UNSUPPORTED;
  if (!root_offsets || !n_selected || (k > 0 && !branch_pos) || (n_tokens > 0 && !delta))
    return HDL_ERR_INVALID_ARG;
  if (!aligned_to(root_offsets, 8) || !aligned_to(n_selected, 4) ||
      (branch_pos && !aligned_to(branch_pos, 4)) || (delta && !aligned_to(delta, 4)) ||
      (branch_delta && !aligned_to(branch_delta, 4)))
    return HDL_ERR_INVALID_ARG;
  const int sms = current_sm_count();
  if (sms <= 0) return HDL_ERR_CUDA;
  cudaStream_t st = as_stream(cuda_stream);
  if (o.min_gap > 0) {
    const int grid = n_roots < 32 * sms ? n_roots : 32 * sms;
    select_spacing_kernel<<<grid, kSelThreads, 0, st>>>(
        delta, valid, n_tokens, root_offsets, n_roots, k, o.min_gap, o.gap_mode, o.lo, o.hi,
        branch_pos, n_selected, branch_delta);
    return launch_status();
  }
  if (k == 0) {
    if (cudaMemsetAsync(n_selected, 0, sizeof(int32_t) * n_roots, st) != cudaSuccess)
      return HDL_ERR_CUDA;
    return HDL_OK;
  }
  const bool vec = aligned_to(delta, 16) && (valid == nullptr || aligned_to(valid, 4));
  return vec ? launch_topk<true>(delta, valid, n_tokens, root_offsets, n_roots, k, o.lo, o.hi,
                                 branch_pos, n_selected, branch_delta, sms, st)
             : launch_topk<false>(delta, valid, n_tokens, root_offsets, n_roots, k, o.lo, o.hi,
                                  branch_pos, n_selected, branch_delta, sms, st);
}
