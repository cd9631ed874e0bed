// Continuation allocation (Section 4.1 "Rollout protocols", Table
// fork-ablation, Section 4.4) and suffix-only loss masks (Section 3.3,
// Eq. branch-sampling).
#include <cuda_runtime.h>

#include <cstdint>
#include <climits>

#include "hdl.h"
#include "hdl_internal.h"

namespace hdl {
namespace {

constexpr int kAssignThreads = 1024;
constexpr int kMaskThreads = 256;

// Rank of the branch point that continuation j (of C) of a root with n
// points branches from: point i gets floor(C/n) + [i < C mod n] consecutive
// continuations (extra to the higher-ranked points), or
// floor(C/n) + [i >= n - C mod n] (extra to the lower-ranked ones).
__device__ __forceinline__ int cont_rank(int j, int C, int n, bool extra_to_higher) {
  const int base = C / n, rem = C % n;
  if (extra_to_higher) {
    const int head = rem * (base + 1);
    return j < head ? j / (base + 1) : rem + (j - head) / base;
  }
  const int head = (n - rem) * base;
  return j < head ? j / base : (n - rem) + (j - head) / (base + 1);
}

// One CTA: an exclusive scan of the continuation counts gives each root's
// first output slot; each thread then fills its root's continuations.
__global__ void __launch_bounds__(kAssignThreads)
    assign_continuations_kernel(const int32_t* __restrict__ n_selected,
                                const int32_t* __restrict__ branch_pos, int32_t n_roots,
                                int32_t k, const int32_t* __restrict__ conts_per_root,
                                int32_t extra_to_higher, int32_t* __restrict__ cont_branch,
                                int64_t capacity) {
  __shared__ int64_t warp_sums[kAssignThreads / 32];
  __shared__ int64_t carry;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < n_roots; base += kAssignThreads) {
    const int r = base + threadIdx.x;
    int64_t C = 0;
    if (r < n_roots) {
      const int32_t c = conts_per_root[r];
      C = c > 0 ? c : 0;
    }
    // inclusive warp scan, then across warps
    int64_t v = C;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int64_t u = __shfl_up_sync(0xffffffffu, v, o);
      if (lane >= o) v += u;
    }
    if (lane == 31) warp_sums[warp] = v;
    __syncthreads();
    if (warp == 0) {
      int64_t w = warp_sums[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int64_t u = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += u;
      }
      warp_sums[lane] = w;
    }
    __syncthreads();
    const int64_t first = carry + (warp > 0 ? warp_sums[warp - 1] : 0) + (v - C);
    if (r < n_roots && C > 0) {
      int n = n_selected[r];
      n = n < 0 ? 0 : (n > k ? k : n);
      for (int j = 0; j < static_cast<int>(C); ++j) {
        const int64_t o = first + j;
        if (o >= capacity) break;
        cont_branch[o] =
            n == 0 ? -1
                   : branch_pos[static_cast<int64_t>(r) * k +
                                cont_rank(j, static_cast<int>(C), n, extra_to_higher != 0)];
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) carry += warp_sums[kAssignThreads / 32 - 1];
    __syncthreads();
  }
}

// 0x01 in every byte of w that is nonzero, 0x00 elsewhere.
__device__ __forceinline__ uint32_t nonzero_bytes(uint32_t w) {
  return (((w & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | w) >> 7 & 0x01010101u;
}

// One warp per continuation c: bytes [s, e) = [offs[c], offs[c+1]) clipped to
// the mask; byte p is on iff p >= thr (= s + b, or never when b < 0) and it is
// valid.  The body, whose vectors start at bytes p with (p + phase) % 16 == 0
// (phase = the mask's address mod 16, the validity bytes' too), is read and
// written 16 bytes per lane, the head and tail bytes one by one, and only the
// one vector that contains thr is resolved byte by byte; four body vectors
// per lane are loaded before any is stored (one at a time measured 5-8 %
// slower).
template <bool kVec>
__global__ void __launch_bounds__(kMaskThreads)
    suffix_mask_kernel(const int32_t* __restrict__ cb, const int64_t* __restrict__ offs,
                       int32_t n_cont, const uint8_t* __restrict__ valid,
                       uint8_t* __restrict__ mask, int64_t mask_len, int32_t phase) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x / 32);
  for (int64_t c = static_cast<int64_t>(blockIdx.x) * (blockDim.x / 32) + (threadIdx.x >> 5);
       c < n_cont; c += warps) {
    int64_t s = offs[c], e = offs[c + 1];
    const int32_t b = cb[c];
    const int64_t thr = b >= 0 ? s + b : INT64_MAX;
    s = s < 0 ? 0 : s;
    e = e > mask_len ? mask_len : e;
    if (e <= s) continue;
    int64_t h = s, body = s;
    if (kVec) {
      h = ((s + phase + 15) & ~int64_t{15}) - phase;
      h = h < e ? h : e;
      body = h + ((e - h) & ~int64_t{15});
    }
    for (int64_t p = s + lane; p < h; p += 32)
      mask[p] = (p >= thr && (valid == nullptr || valid[p] != 0)) ? 1 : 0;
    // body: four 16-byte vectors per lane in flight, then their stores
    constexpr int kU = 4;
    auto finish = [&](uint4 v, int64_t p) {
      if (valid) {
        v.x = nonzero_bytes(v.x);
        v.y = nonzero_bytes(v.y);
        v.z = nonzero_bytes(v.z);
        v.w = nonzero_bytes(v.w);
      }
      if (p + 16 <= thr) {
        v = make_uint4(0u, 0u, 0u, 0u);
      } else if (p < thr) {
        uint8_t* vb = reinterpret_cast<uint8_t*>(&v);
#pragma unroll
        for (int i = 0; i < 16; ++i)
          if (p + i < thr) vb[i] = 0;
      }
      *reinterpret_cast<uint4*>(mask + p) = v;
    };
    const uint4 ones = make_uint4(0x01010101u, 0x01010101u, 0x01010101u, 0x01010101u);
    int64_t p = h + 16 * lane;
    for (; p + 16 * 32 * (kU - 1) < body; p += 16 * 32 * kU) {
      uint4 v[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u)
        v[u] = valid ? *reinterpret_cast<const uint4*>(valid + p + 16 * 32 * u) : ones;
#pragma unroll
      for (int u = 0; u < kU; ++u) finish(v[u], p + 16 * 32 * u);
    }
    for (; p < body; p += 16 * 32)
      finish(valid ? *reinterpret_cast<const uint4*>(valid + p) : ones, p);
    for (int64_t p = body + lane; p < e; p += 32)
      mask[p] = (p >= thr && (valid == nullptr || valid[p] != 0)) ? 1 : 0;
  }
}

}  // namespace
}  // namespace hdl

using namespace hdl;

extern "C" hdl_status hdl_assign_continuations(const int32_t* n_selected,
                                               const int32_t* branch_pos, int32_t n_roots,
                                               int32_t k, const int32_t* conts_per_root,
                                               int32_t extra_to_higher, int32_t* cont_branch,
                                               int64_t n_cont_capacity, void* cuda_stream) {
  HostRange range_("hdl_assign_continuations");
  if (n_roots < 0 || k < 0 || n_cont_capacity < 0) return HDL_ERR_INVALID_ARG;
  if (k > 16) return HDL_ERR_UNSUPPORTED;
  if (n_roots == 0 || n_cont_capacity == 0) return HDL_OK;
  if (!n_selected || !conts_per_root || !cont_branch || (k > 0 && !branch_pos))
    return HDL_ERR_INVALID_ARG;
  if (!aligned_to(n_selected, 4) || !aligned_to(conts_per_root, 4) ||
      !aligned_to(cont_branch, 4) || (branch_pos && !aligned_to(branch_pos, 4)))
    return HDL_ERR_INVALID_ARG;
  assign_continuations_kernel<<<1, kAssignThreads, 0, as_stream(cuda_stream)>>>(
      n_selected, branch_pos, n_roots, k, conts_per_root, extra_to_higher, cont_branch,
      n_cont_capacity);
  return launch_status();
}

extern "C" hdl_status hdl_suffix_mask(const int32_t* cont_branch, const int64_t* cont_offsets,
                                      int32_t n_cont, const uint8_t* cont_valid, uint8_t* mask,
                                      int64_t mask_len, void* cuda_stream) {
  HostRange range_("hdl_suffix_mask");
  if (n_cont < 0 || mask_len < 0) return HDL_ERR_INVALID_ARG;
  if (n_cont == 0 || mask_len == 0) return HDL_OK;
  if (!cont_branch || !cont_offsets || !mask) return HDL_ERR_INVALID_ARG;
  if (!aligned_to(cont_branch, 4) || !aligned_to(cont_offsets, 8)) return HDL_ERR_INVALID_ARG;
  // 16-byte vectors wherever the mask's and validity bytes' alignments agree
  const int phase = static_cast<int>(reinterpret_cast<uintptr_t>(mask) & 15u);
  const bool vec = cont_valid == nullptr ||
                   static_cast<int>(reinterpret_cast<uintptr_t>(cont_valid) & 15u) == phase;
  const int sms = current_sm_count();
  if (sms <= 0) return HDL_ERR_CUDA;
  const int64_t blocks = ceil_div(n_cont, kMaskThreads / 32);   // one warp per continuation
  const int grid = static_cast<int>(blocks < 16 * sms ? blocks : 16 * sms);
  cudaStream_t st = as_stream(cuda_stream);
  if (vec)
    suffix_mask_kernel<true><<<grid, kMaskThreads, 0, st>>>(cont_branch, cont_offsets, n_cont,
                                                            cont_valid, mask, mask_len, phase);
  else
    suffix_mask_kernel<false><<<grid, kMaskThreads, 0, st>>>(cont_branch, cont_offsets, n_cont,
                                                             cont_valid, mask, mask_len, phase);
  return launch_status();
}
