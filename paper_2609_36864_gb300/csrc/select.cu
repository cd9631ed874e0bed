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
// 16-byte loads (4 scores + 4 validity bytes per lane, a batch of 512
// positions per warp) into one exact top-k list per warp held across its
// lanes.  The first batch of a slice sets a floor on the k-th best score (the
// k-th largest of the 32 lane maxima); after that a batch costs a max over
// each lane's 16 scores and one warp vote unless some score reaches the
// threshold.  The few candidates that beat the current k-th best (about
// k ln(T/k) per root) are inserted one after the other (ballot + shift), or,
// when many arrive together, by a bitonic sort of the warp's 32 candidates
// and a bitonic merge with the list.  Many roots: S warps per root (usually
// 1) in a persistent grid; few roots: 16 warps per root; the partial lists
// of a root's warps are merged pairwise, a bitonic merge per level.
// Spacing rule (Section 4.4; min_gap > 0, |t - a| < min_gap counts as too
// close):
//   drop-lower (gap_mode 1): the plain top-k above, then the root's warp walks
//     its k points in rank order and drops each one too close to a kept one;
//   greedy (gap_mode 0): the greedy walk of the ranked list accepts, in
//     rank order, each candidate not too close to an accepted one.  The same
//     streaming kernel collects the 16 best candidates far enough from every
//     point accepted so far, the root's warp walks them in rank order, and a
//     new pass follows only while fewer than k are accepted and the pass came
//     back full -- one to three passes on clustered scores, k at most.
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdlib>

#include "hdl.h"
#include "hdl_internal.h"

namespace hdl {
namespace {

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

// The warp's running top-k is distributed over its lanes: lane j < k holds
// the j-th best key so far (0 = empty), lanes >= k hold 0.  tau = lane k-1's
// key is the exact k-th best; a candidate must beat it to enter.
struct WarpTopK {
  uint64_t mine;   // this lane's entry
  uint64_t tau;    // k-th best so far, on every lane
  float tau_s;     // score a candidate must reach: max(tau's score, floor)
  float floor;     // a lower bound on the final k-th best score (-inf: none)
};

// Inverse of score_order on a key's high word.
__device__ __forceinline__ float key_score(uint64_t key) {
  if (key == 0ull) return -INFINITY;
  const uint32_t u = static_cast<uint32_t>(key >> 32);
  return __uint_as_float((u & 0x80000000u) ? (u ^ 0x80000000u) : ~u);
}

// Bitonic network over the warp, one 64-bit key per lane.  One
// compare-exchange with the lane `stride` away: the lower lane of the pair
// keeps the larger key when keep_max.
__device__ __forceinline__ uint64_t cmpx(uint64_t x, int stride, bool keep_max) {
  const uint64_t y = __shfl_xor_sync(0xffffffffu, x, stride);
  return keep_max == (x > y) ? x : y;
}

// Sort the warp's 32 keys into descending lane order.
__device__ __forceinline__ uint64_t warp_sort_desc(uint64_t x, int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1)
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      // blocks of `size` lanes alternate descending / ascending, so that
      // each pair of neighbouring blocks forms a bitonic sequence
      const bool desc = (lane & size) == 0;
      const bool lower = (lane & stride) == 0;
      x = cmpx(x, stride, lower == desc);
    }
  return x;
}

// Merge two descending lists of at most 16 keys, a (in lanes 0..15) and b
// (lane j of b_rev holds b[31 - j], so lanes 16..31 read b reversed): the
// 32 values form a bitonic sequence and five half-cleaner steps sort it.
// Returns the merged list, descending, in lanes 0..31.
__device__ __forceinline__ uint64_t bitonic_merge16(uint64_t a, uint64_t b_rev, int lane) {
  uint64_t x = lane < 16 ? a : b_rev;
#pragma unroll
  for (int stride = 16; stride > 0; stride >>= 1) x = cmpx(x, stride, (lane & stride) == 0);
  return x;
}

__device__ __forceinline__ void wtk_set(WarpTopK& w, uint64_t merged, int k, int lane) {
  w.mine = lane < k ? merged : 0ull;
  w.tau = __shfl_sync(0xffffffffu, w.mine, k - 1);
  w.tau_s = fmaxf(key_score(w.tau), w.floor);
}

// Offer one key per lane (0 = none): the keys that beat the k-th best are
// inserted -- one after the other in lane order when there are few, by
// sorting the warp's keys and merging the top 16 with the list when there
// are many.  In the one-by-one case no key is re-tested after an insertion:
// inserting a key that no longer beats the k-th best changes nothing (its
// slot is k, which is cleared), so the candidates' shuffles do not wait on
// the list and the chain per insertion is one ballot and one shift.
constexpr int kBulkMin = 12;

__device__ __forceinline__ void wtk_offer_key(WarpTopK& w, uint64_t key, int k, int lane) {
  unsigned pending = __ballot_sync(0xffffffffu, key > w.tau);
  if (!pending) return;
  if (__popc(pending) >= kBulkMin) {
    const uint64_t c = warp_sort_desc(key > w.tau ? key : 0ull, lane);
    const uint64_t c_rev = __shfl_sync(0xffffffffu, c, 31 - lane);
    wtk_set(w, bitonic_merge16(w.mine, c_rev, lane), k, lane);
    return;
  }
  do {
    const int src = __ffs(pending) - 1;
    pending &= pending - 1u;
    const uint64_t cand = __shfl_sync(0xffffffffu, key, src);
    const int pos = __popc(__ballot_sync(0xffffffffu, w.mine > cand));
    const uint64_t prev = __shfl_up_sync(0xffffffffu, w.mine, 1);
    if (lane > pos) w.mine = prev;
    if (lane == pos) w.mine = cand;
    if (lane >= k) w.mine = 0ull;
  } while (pending);
  w.tau = __shfl_sync(0xffffffffu, w.mine, k - 1);
  w.tau_s = fmaxf(key_score(w.tau), w.floor);
}

// Which root positions may enter a list: any (plain top-k), or, for the
// greedy spacing rule, only those at least min_gap away from every point
// accepted so far (the accepted list is the same on every lane).
struct AnyPos {
  static constexpr bool kAll = true;
  __device__ __forceinline__ bool ok(int32_t) const { return true; }
};

struct FarFromAccepted {
  static constexpr bool kAll = false;
  const int32_t* acc;   // the group's accepted root positions (shared memory)
  int na;
  int32_t gap;
  __device__ __forceinline__ bool ok(int32_t t) const {
    for (int i = 0; i < na; ++i) {
      const int32_t dd = t - acc[i];
      if ((dd < 0 ? -dd : dd) < gap) return false;
    }
    return true;
  }
};

// Offer each lane's candidate (score s at root position t; ok = valid): a
// candidate whose score is below the k-th best's cannot beat it and is
// rejected by the float compare alone; the others get their key built (NaN
// scores never pass the compare).
template <class F>
__device__ __forceinline__ void wtk_offer(WarpTopK& w, float s, bool ok, int64_t t, int k,
                                          int lane, const F& f) {
  ok = ok && s >= w.tau_s && f.ok(static_cast<int32_t>(t));
  if (!__any_sync(0xffffffffu, ok)) return;
  wtk_offer_key(w, ok ? make_key(s, t) : 0ull, k, lane);
}

// One warp-wide batch of the vector body: kBatch groups of 32 x 4
// consecutive positions (16 bytes of scores and 4 validity bytes per lane
// per group); positions at or past `body` read as invalid.
constexpr int kBatch = 4;
constexpr int32_t kSpan = 4 * 32 * kBatch;   // positions per batch

struct Batch {
  float4 d[kBatch];
  uint32_t v[kBatch];
};

// Positions are int32 inside the streaming loops (the entry point rejects
// n_tokens >= 2^31).  A full batch (q + kSpan <= body) loads unguarded.
template <bool kFull>
__device__ __forceinline__ void load_batch(Batch& b, const float* delta, const uint8_t* valid,
                                           int32_t q, int32_t body, int lane) {
#pragma unroll
  for (int i = 0; i < kBatch; ++i) {
    const int32_t p = q + 4 * (32 * i + lane);
    if (kFull || p < body) {
      b.d[i] = *reinterpret_cast<const float4*>(delta + p);
      b.v[i] = valid ? *reinterpret_cast<const uint32_t*>(valid + p) : 0x01010101u;
    } else {
      b.d[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      b.v[i] = 0u;
    }
  }
}

// Examine a batch whose first position is q (absolute; root position =
// absolute - start).  The common case costs a max over the lane's 16 scores
// and one vote: no score reaches the threshold, so nothing can enter.
// Otherwise the lanes' passing valid candidates are offered in rounds, each
// lane its next one per round, until no lane has any left.
template <class F>
__device__ __forceinline__ void offer_batch(WarpTopK& w, const Batch& b, const float* delta,
                                            int32_t q, int32_t start, int k, int lane,
                                            const F& f) {
  float mx = -INFINITY;   // fmaxf ignores NaN scores
#pragma unroll
  for (int i = 0; i < kBatch; ++i)
    mx = fmaxf(mx, fmaxf(fmaxf(b.d[i].x, b.d[i].y), fmaxf(b.d[i].z, b.d[i].w)));
  if (!__any_sync(0xffffffffu, mx >= w.tau_s)) return;
  uint32_t pass = 0;   // bit 4i+c: component c of group i
#pragma unroll
  for (int i = 0; i < kBatch; ++i) {
    pass |= static_cast<uint32_t>((b.v[i] & 0xFFu) != 0 && b.d[i].x >= w.tau_s) << (4 * i);
    pass |= static_cast<uint32_t>((b.v[i] & 0xFF00u) != 0 && b.d[i].y >= w.tau_s) << (4 * i + 1);
    pass |= static_cast<uint32_t>((b.v[i] & 0xFF0000u) != 0 && b.d[i].z >= w.tau_s)
            << (4 * i + 2);
    pass |= static_cast<uint32_t>((b.v[i] & 0xFF000000u) != 0 && b.d[i].w >= w.tau_s)
            << (4 * i + 3);
  }
  while (__any_sync(0xffffffffu, pass != 0)) {
    const int j = pass ? __ffs(pass) - 1 : -1;
    pass &= pass - 1u;
    // the candidate's score, read again from the batch just loaded (a cache
    // hit; cheaper in instructions than selecting it among 16 registers)
    const int32_t p = q + 4 * (32 * (j >> 2) + lane) + (j & 3);
    const float sj = j >= 0 ? delta[p] : -INFINITY;
    const int32_t t = p - start;
    wtk_offer_key(w, j >= 0 && sj >= w.tau_s && f.ok(t) ? make_key(sj, t) : 0ull, k, lane);
  }
}

// Sort 32 floats (one per lane) into descending lane order.
__device__ __forceinline__ float warp_sort_desc_f(float x, int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1)
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const float y = __shfl_xor_sync(0xffffffffu, x, stride);
      const bool keep_max = ((lane & stride) == 0) == ((lane & size) == 0);
      x = keep_max ? fmaxf(x, y) : fminf(x, y);
    }
  return x;
}

// A floor for the k-th best score from a warp's first batch: among the 32
// lane maxima (the best valid candidate of each lane), the k-th largest is
// reached by at least k distinct candidates, so no score below it can be
// among the k best of the slice.  Candidates below it are then rejected by
// the float compare alone, which spares most of the insertions a root
// otherwise pays while its list fills.
// Under a position filter a lane contributes its best valid candidate only
// if the filter admits it (else -inf): the k-th largest contribution is
// still reached by k distinct admitted candidates.
template <class F>
__device__ __forceinline__ void set_floor(WarpTopK& w, const Batch& b, int32_t q, int32_t start,
                                          int k, int lane, const F& f) {
  float m = -INFINITY;   // fmaxf ignores a NaN operand
  if constexpr (F::kAll) {
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
      m = fmaxf(m, (b.v[i] & 0xFFu) != 0 ? b.d[i].x : -INFINITY);
      m = fmaxf(m, (b.v[i] & 0xFF00u) != 0 ? b.d[i].y : -INFINITY);
      m = fmaxf(m, (b.v[i] & 0xFF0000u) != 0 ? b.d[i].z : -INFINITY);
      m = fmaxf(m, (b.v[i] & 0xFF000000u) != 0 ? b.d[i].w : -INFINITY);
    }
  } else {
    int32_t at = 0;   // position of the lane's best (NaN never compares greater)
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
      const int32_t t = q + 4 * (32 * i + lane) - start;
      const float c[4] = {b.d[i].x, b.d[i].y, b.d[i].z, b.d[i].w};
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (((b.v[i] >> (8 * j)) & 0xFFu) != 0 && c[j] > m) {
          m = c[j];
          at = t + j;
        }
    }
    if (!f.ok(at)) m = -INFINITY;
  }
  m = warp_sort_desc_f(m, lane);
  w.floor = fmaxf(w.floor, __shfl_sync(0xffffffffu, m, k - 1));
  w.tau_s = fmaxf(w.tau_s, w.floor);
}

// The warp streams absolute positions [a0, a1) of the root starting at
// `start`: a vector body walked in warp-uniform batches (all loads of a
// batch issued before any is used; the first batch sets the floor), then the
// scalar head and tail.
template <bool kVec, class F>
__device__ __forceinline__ void stream_range(WarpTopK& w, const float* delta, const uint8_t* valid,
                                             int64_t start64, int64_t a0_64, int64_t a1_64, int k,
                                             int lane, int phase, const F& f) {
  const int32_t start = static_cast<int32_t>(start64);
  const int32_t a0 = static_cast<int32_t>(a0_64), a1 = static_cast<int32_t>(a1_64);
  if (!kVec) {
    for (int32_t q = a0; q < a1; q += 32) {
      const int32_t p = q + lane;
      const bool in = p < a1;
      wtk_offer(w, in ? delta[p] : 0.f, in && (valid == nullptr || valid[p] != 0), p - start, k,
                lane, f);
    }
    return;
  }
  // vector positions q have (q + phase) % 4 == 0: delta + q is 16-byte and
  // valid + q 4-byte aligned
  const int32_t up = a0 + ((4 - ((a0 + phase) & 3)) & 3);
  const int32_t h = up < a1 ? up : a1;
  const int32_t body = h + ((a1 - h) & ~3);
  for (int32_t q = h; q < body; q += kSpan) {
    Batch x;
    if (q + kSpan <= body)
      load_batch<true>(x, delta, valid, q, body, lane);
    else
      load_batch<false>(x, delta, valid, q, body, lane);
    if (q == h) set_floor(w, x, q, start, k, lane, f);
    offer_batch(w, x, delta, q, start, k, lane, f);
  }
  // scalar head and tail (at most 3 positions each)
  const int32_t p = lane < 4 ? a0 + lane : body + (lane - 4);
  const bool in = lane < 4 ? p < h : p < a1;
  wtk_offer(w, in ? delta[p] : 0.f, in && (valid == nullptr || valid[p] != 0), p - start, k,
            lane, f);
}

// Drop-lower spacing on a finished list (lanes 0..n-1, best first): in rank
// order, a point within min_gap of a kept higher-ranked point is dropped;
// the kept ones are packed to the front in rank order and n becomes their
// count.
__device__ __forceinline__ void drop_close(WarpTopK& w, int& n, int32_t min_gap, int lane) {
  const int32_t t_me = static_cast<int32_t>(key_pos(w.mine));
  bool keep = lane < n;
  for (int i = 1; i < n; ++i) {
    const int32_t t_i = __shfl_sync(0xffffffffu, t_me, i);
    const int32_t dd = t_me - t_i;
    const bool close = keep && lane < i && (dd < 0 ? -dd : dd) < min_gap;
    if (__any_sync(0xffffffffu, close) && lane == i) keep = false;
  }
  const unsigned kept = __ballot_sync(0xffffffffu, keep);
  uint64_t out = 0ull;
  int j = 0;
  for (int i = 0; i < n; ++i) {
    const uint64_t ki = __shfl_sync(0xffffffffu, w.mine, i);
    if ((kept >> i) & 1u) {
      if (lane == j) out = ki;
      ++j;
    }
  }
  w.mine = out;
  n = j;
}

// S warps share a root: S = 1, 2, 4, 8 in blocks of 8 warps (8/S roots at a
// time per block), S = 16 in blocks of 16 warps.
template <int S>
struct TopkShape {
  static constexpr int kWarps = S == 16 ? 16 : 8;    // warps per block
  static constexpr int kGroups = kWarps / S;         // roots in flight per block
  static constexpr int kMinBlocks = S == 16 ? 1 : (S == 1 ? 5 : 4);
};

__device__ __forceinline__ void group_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// One pass of a root's group of S warps: every warp streams its slice of
// [a0, a1) into a list of kk entries (positions the filter admits only),
// then, for S > 1, the lists are merged pairwise into the first warp's
// through shared memory (a bitonic merge per level, the group's own named
// barrier between levels).  Returns true on the warp that holds the result.
template <int S, bool kVec, class F>
__device__ __forceinline__ bool collect(WarpTopK& w, uint64_t (*lists)[32], const float* delta,
                                        const uint8_t* valid, int64_t start, int64_t a0,
                                        int64_t a1, int kk, int lane, int warp, int grp, int ws,
                                        int phase, const F& f) {
  w = WarpTopK{0ull, 0ull, -INFINITY, -INFINITY};
  if constexpr (S == 1) {
    if (a1 > a0) stream_range<kVec>(w, delta, valid, start, a0, a1, kk, lane, phase, f);
    return true;
  } else {
    const int64_t len = a1 > a0 ? a1 - a0 : 0;
    const int64_t per = ((len + S - 1) / S + 3) & ~int64_t{3};
    const int64_t s0 = a0 + per * ws;
    const int64_t s1 = s0 + per < a1 ? s0 + per : a1;
    if (s0 < s1) stream_range<kVec>(w, delta, valid, start, s0, s1, kk, lane, phase, f);
    lists[warp][lane] = w.mine;
    const int bar = 1 + grp, nthreads = 32 * S;
    group_sync(bar, nthreads);
#pragma unroll
    for (int half = S / 2; half >= 1; half >>= 1) {
      if (ws < half) {
        const uint64_t m =
            bitonic_merge16(lists[warp][lane & 15], lists[warp + half][(31 - lane) & 15], lane);
        w.mine = lane < kk ? m : 0ull;
        lists[warp][lane] = w.mine;
      }
      group_sync(bar, nthreads);
    }
    return ws == 0;
  }
}

enum SelectMode : int { kPlain = 0, kDropLower = 1, kGreedy = 2 };

// kMode: plain top-k; drop-lower spacing applied to the finished list; or
// greedy spacing -- passes that each collect the kMaxK best positions far
// enough from every point accepted so far and walk them in rank order,
// accepting those still far enough, until k are accepted or a pass comes
// back short (no candidate left).  Every pass but the last accepts at least
// its first entry, so there are at most k passes; usually one to three.
template <int S, bool kVec, int kMode>
__global__ void __launch_bounds__(32 * TopkShape<S>::kWarps, TopkShape<S>::kMinBlocks)
    select_topk_kernel(const float* __restrict__ delta, const uint8_t* __restrict__ valid,
                       int64_t n_tokens, const int64_t* __restrict__ root_offsets,
                       int32_t n_roots, int32_t k, int32_t lo, int32_t hi, int32_t min_gap,
                       int32_t phase, int32_t* __restrict__ branch_pos,
                       int32_t* __restrict__ n_selected, float* __restrict__ branch_delta) {
  using Sh = TopkShape<S>;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int grp = warp / S, ws = warp % S;
  __shared__ uint64_t lists[S == 1 ? 1 : Sh::kWarps][32];
  // greedy: the group's accepted positions, then their count and whether
  // the root is done (written by the warp that walks each pass's list)
  __shared__ int32_t accepted[kMode == kGreedy ? Sh::kGroups : 1][kMaxK + 2];
  const int64_t step = static_cast<int64_t>(gridDim.x) * Sh::kGroups;
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * Sh::kGroups + grp; r < n_roots; r += step) {
    const int64_t start = root_offsets[r];
    const int64_t end = root_offsets[r + 1];
    const int64_t T = end > start ? end - start : 0;
    const int64_t w_lo = lo > 0 ? lo : 0;
    const int64_t w_hi = hi <= 0 ? T : (hi < T ? hi : T);
    int64_t a0 = start + w_lo, a1 = start + w_hi;
    if (a0 < 0) a0 = 0;
    if (a1 > n_tokens) a1 = n_tokens;
    WarpTopK w;
    if constexpr (kMode != kGreedy) {
      if (!collect<S, kVec>(w, lists, delta, valid, start, a0, a1, k, lane, warp, grp, ws, phase,
                            AnyPos{}))
        continue;
      int n = __popc(__ballot_sync(0xffffffffu, w.mine != 0ull));
      if constexpr (kMode == kDropLower) {
        if (n > 1) drop_close(w, n, min_gap, lane);
      }
      if (lane < k) {
        const int64_t o = r * k + lane;
        if (lane < n) {
          const int64_t t = key_pos(w.mine);
          branch_pos[o] = static_cast<int32_t>(t);
          // the key holds the absolute position minus the root start, mod 2^32
          if (branch_delta)
            branch_delta[o] = delta[static_cast<uint32_t>(start) + static_cast<uint32_t>(t)];
        } else {
          branch_pos[o] = -1;
          if (branch_delta) branch_delta[o] = __int_as_float(0x7fc00000);
        }
      }
      if (lane == 0) n_selected[r] = n;
    } else {
      int32_t* acc = accepted[grp];
      FarFromAccepted far{acc, 0, min_gap};
      bool holder = false;
      for (;;) {
        holder = collect<S, kVec>(w, lists, delta, valid, start, a0, a1, kMaxK, lane, warp, grp,
                                  ws, phase, far);
        bool done = false;
        if (holder) {
          // every entry is far enough from the points accepted before this
          // pass, so walking them in rank order is the drop-lower rule on
          // the list: keep those not too close to a kept better one, and
          // accept the first ones kept until k are accepted
          const int m = __popc(__ballot_sync(0xffffffffu, w.mine != 0ull));
          int kept = m;
          if (kept > 1) drop_close(w, kept, min_gap, lane);
          const int take = kept < k - far.na ? kept : k - far.na;
          if (lane < take) acc[far.na + lane] = static_cast<int32_t>(key_pos(w.mine));
          far.na += take;
          done = far.na >= k || m < kMaxK;
          if (lane == 0) {
            acc[kMaxK] = far.na;
            acc[kMaxK + 1] = done;
          }
        }
        if constexpr (S > 1) {
          group_sync(1 + grp, 32 * S);
          far.na = acc[kMaxK];
          done = acc[kMaxK + 1] != 0;
        } else {
          __syncwarp();
        }
        if (done) break;
      }
      if (!holder) continue;
      if (lane < k) {
        const int64_t o = r * k + lane;
        const bool have = lane < far.na;
        const int32_t pos = have ? acc[lane] : -1;
        branch_pos[o] = pos;
        if (branch_delta)
          branch_delta[o] = have ? delta[static_cast<uint32_t>(start) + static_cast<uint32_t>(pos)]
                                 : __int_as_float(0x7fc00000);
      }
      if (lane == 0) n_selected[r] = far.na;
    }
  }
}

// HDL_SELECT_SPLIT (1, 2, 4 or 8) fixes the warps per root of the many-roots
// mode, for tests and tuning; results do not depend on it.
int select_split_override() {
  static const int v = [] {
    const char* e = std::getenv("HDL_SELECT_SPLIT");
    if (e && (e[0] == '1' || e[0] == '2' || e[0] == '4' || e[0] == '8') && e[1] == '\0')
      return e[0] - '0';
    return 0;
  }();
  return v;
}

// Arguments of one selection launch (the kernel parameters after the grid).
struct SelectArgs {
  const float* delta;
  const uint8_t* valid;
  int64_t n_tokens;
  const int64_t* offs;
  int32_t n_roots, k, lo, hi, gap;
  int32_t phase;   // (delta address / 4) mod 4; valid's address has the same residue mod 4
  int32_t* bp;
  int32_t* ns;
  float* bd;
};

template <int S, bool kVec, int kMode>
hdl_status launch_topk_s(const SelectArgs& a, int grid, cudaStream_t st) {
  select_topk_kernel<S, kVec, kMode><<<grid, 32 * TopkShape<S>::kWarps, 0, st>>>(
      a.delta, a.valid, a.n_tokens, a.offs, a.n_roots, a.k, a.lo, a.hi, a.gap, a.phase, a.bp,
      a.ns, a.bd);
  return launch_status();
}

// Few roots (< 2 per SM): 16 warps per root, one block each, so that every
// root is done in a single short pass.  Many roots: a persistent grid of
// 8-warp blocks; S warps per root, S the smallest power of two that gives
// every resident warp a slice (so that a few hundred long roots still keep
// enough loads in flight), but no slice shorter than 1024 positions.  (More
// slices than that only add per-slice work: 8192 roots of 4096 positions
// took 47, 51, 67 and 84 us at S = 1, 2, 4, 8.  At S = 1 the kernel runs
// within 8% of a read-only kernel with the same one-warp-per-root pattern
// and occupancy; neither deeper register prefetch nor a shared-memory ring
// filled by bulk copies made it faster.)  kMode selects the spacing rule,
// with min_gap = a.gap.
template <bool kVec, int kMode>
hdl_status launch_topk(const SelectArgs& a, int sms, cudaStream_t st) {
  if (a.n_roots < 2 * sms) return launch_topk_s<16, kVec, kMode>(a, a.n_roots, st);
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, select_topk_kernel<1, kVec, kMode>,
                                                    256, 0) != cudaSuccess || per_sm <= 0)
    per_sm = 4;
  const int64_t resident_warps = static_cast<int64_t>(per_sm) * 8 * sms;
  int64_t span = a.n_tokens / a.n_roots;
  if (a.hi > 0 && a.hi < span) span = a.hi;
  span -= a.lo > 0 ? a.lo : 0;
  int S = 1;
  while (S < 8 && int64_t{a.n_roots} * S < resident_warps && span / (2 * S) >= 1024) S *= 2;
  if (const int forced = select_split_override()) S = forced;
  const int64_t blocks = (int64_t{a.n_roots} * S + 7) / 8;
  const int64_t cap = static_cast<int64_t>(per_sm) * sms;
  const int grid = static_cast<int>(blocks < cap ? blocks : cap);
  switch (S) {
    case 1: return launch_topk_s<1, kVec, kMode>(a, grid, st);
    case 2: return launch_topk_s<2, kVec, kMode>(a, grid, st);
    case 4: return launch_topk_s<4, kVec, kMode>(a, grid, st);
    default: return launch_topk_s<8, kVec, kMode>(a, grid, st);
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
  HostRange range_("hdl_select_branches");
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
  if (k == 0) {
    if (cudaMemsetAsync(n_selected, 0, sizeof(int32_t) * n_roots, st) != cudaSuccess)
      return HDL_ERR_CUDA;
    return HDL_OK;
  }
  // 16-byte vectors wherever the scores' and validity bytes' alignments agree
  // (buffers sliced at the same token offset included)
  const int phase = static_cast<int>((reinterpret_cast<uintptr_t>(delta) >> 2) & 3u);
  const bool vec = valid == nullptr ||
                   static_cast<int>(reinterpret_cast<uintptr_t>(valid) & 3u) == phase;
  const SelectArgs a{delta, valid, n_tokens, root_offsets, n_roots, k, o.lo, o.hi, o.min_gap,
                     phase, branch_pos, n_selected, branch_delta};
  if (o.min_gap > 0 && o.gap_mode == 0)
    return vec ? launch_topk<true, kGreedy>(a, sms, st) : launch_topk<false, kGreedy>(a, sms, st);
  if (o.min_gap > 0)
    return vec ? launch_topk<true, kDropLower>(a, sms, st)
               : launch_topk<false, kDropLower>(a, sms, st);
  return vec ? launch_topk<true, kPlain>(a, sms, st) : launch_topk<false, kPlain>(a, sms, st);
}
