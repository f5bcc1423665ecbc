// Table 2 Q4: the key self-join A.id = B.id AND A.review_id < B.review_id over
// the selected rows, materialised on the device as (a, b) row pairs so that
// only the table crosses PCIe (O(N) rather than the O(N^2) pairs, §4.3).
//
// The candidates' keys are sorted with a stable LSD radix sort (8-bit digits,
// 8 passes over the 64-bit key; the payload is the candidate's index, so each
// key group lists its rows in ascending order).  Group heads, a scan over
// them and each candidate's pair count (the group members after it) give the
// pair offsets in candidate order, and every candidate then writes its pairs:
// the result is in ascending (a, b) order.
#include <utility>

#include "common.cuh"
#include "kernels.h"

namespace aiq {
namespace {

constexpr int kSortThreads = 256;
constexpr int kSortItems = 8;                             // per thread
constexpr int kSortTile = kSortThreads * kSortItems;       // 2048 keys per block
constexpr int kRadix = 256;

__device__ __forceinline__ int digit_of(uint64_t k, int shift) { return static_cast<int>((k >> shift) & 0xFF); }

// hist[d * n_blocks + b] = keys of block b whose digit is d.
__global__ void __launch_bounds__(kSortThreads) k_radix_hist(const uint64_t* keys, int64_t n, int shift,
                                                             int32_t* hist, int64_t n_blocks) {
  __shared__ int h[kRadix];
  h[threadIdx.x] = 0;
  __syncthreads();
  const int64_t base = static_cast<int64_t>(blockIdx.x) * kSortTile;
#pragma unroll
  for (int j = 0; j < kSortItems; ++j) {
    const int64_t i = base + j * kSortThreads + threadIdx.x;
    if (i < n) atomicAdd(&h[digit_of(keys[i], shift)], 1);
  }
  __syncthreads();
  hist[static_cast<int64_t>(threadIdx.x) * n_blocks + blockIdx.x] = h[threadIdx.x];
}

// Stable scatter: item i of the tile goes to offsets[digit][block] + (items of
// the same digit before it in the tile).  The tile is walked in 8 rounds of
// 256 consecutive items; within a round the rank comes from the warp's
// match mask and the counts of the warps before it.
__global__ void __launch_bounds__(kSortThreads) k_radix_scatter(const uint64_t* keys_in, const int32_t* vals_in,
                                                                int64_t n, int shift, const int64_t* offsets,
                                                                int64_t n_blocks, uint64_t* keys_out,
                                                                int32_t* vals_out) {
  constexpr int NW = kSortThreads / 32;
  __shared__ int64_t base_off[kRadix];
  __shared__ int warp_cnt[NW][kRadix];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  base_off[threadIdx.x] = offsets[static_cast<int64_t>(threadIdx.x) * n_blocks + blockIdx.x];
  const int64_t tile0 = static_cast<int64_t>(blockIdx.x) * kSortTile;
  for (int j = 0; j < kSortItems; ++j) {
    for (int w = 0; w < NW; ++w) warp_cnt[w][threadIdx.x] = 0;
    __syncthreads();
    const int64_t i = tile0 + j * kSortThreads + threadIdx.x;
    const bool live = i < n;
    const uint64_t k = live ? keys_in[i] : 0ull;
    const int d = live ? digit_of(k, shift) : kRadix;  // kRadix: a lane without an item
    const unsigned peers = __match_any_sync(0xffffffffu, d);
    const int rank = __popc(peers & ((1u << lane) - 1u));
    if (live && rank == 0) warp_cnt[warp][d] = __popc(peers);
    __syncthreads();
    if (live) {
      int before = 0;
      for (int w = 0; w < warp; ++w) before += warp_cnt[w][d];
      const int64_t dst = base_off[d] + before + rank;
      keys_out[dst] = k;
      vals_out[dst] = vals_in[i];
    }
    __syncthreads();
    int total = 0;
    for (int w = 0; w < NW; ++w) total += warp_cnt[w][threadIdx.x];
    base_off[threadIdx.x] += total;
    __syncthreads();
  }
}

__global__ void k_gather_keys(const int64_t* col, const int32_t* ids, int64_t n, uint64_t* keys, int32_t* vals) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= n) return;
  keys[i] = static_cast<uint64_t>(col[ids[i]]);
  vals[i] = static_cast<int32_t>(i);
}

__global__ void k_group_heads(const uint64_t* keys, int64_t n, int32_t* heads) {
  const int64_t p = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (p >= n) return;
  heads[p] = p == 0 || keys[p] != keys[p - 1];
}

// group_start[g] = sorted position of group g's first member; group_start[G] = n.
__global__ void k_group_starts(const int32_t* heads, const int64_t* head_excl, int64_t n, int64_t* group_start) {
  const int64_t p = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (p >= n) return;
  if (heads[p]) group_start[head_excl[p]] = p;
  if (p == n - 1) group_start[head_excl[p] + heads[p]] = n;
}

// Pairs of each candidate (in candidate order): the members of its group after it.
__global__ void k_pair_counts(const int32_t* sorted_idx, const int32_t* heads, const int64_t* head_excl,
                              const int64_t* group_start, int64_t n, int32_t* counts) {
  const int64_t p = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (p >= n) return;
  const int64_t g = head_excl[p] + heads[p] - 1;
  counts[sorted_idx[p]] = static_cast<int32_t>(group_start[g + 1] - p - 1);
}

__global__ void k_emit_pairs(const int32_t* sorted_idx, const int32_t* counts, const int64_t* pair_off,
                             const int32_t* ids, int64_t n, int32_t* pa, int32_t* pb) {
  const int64_t p = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (p >= n) return;
  const int32_t ci = sorted_idx[p];
  const int32_t a = ids[ci];
  const int32_t cnt = counts[ci];
  const int64_t at = pair_off[ci];
  for (int32_t k = 1; k <= cnt; ++k) {
    pa[at + k - 1] = a;
    pb[at + k - 1] = ids[sorted_idx[p + k]];
  }
}

inline unsigned blocks_of(int64_t n, int per) { return static_cast<unsigned>((n + per - 1) / per); }

}  // namespace

void launch_self_join_pairs_plan(const int64_t* key_col, const int32_t* ids, int64_t S, const SelfJoinScratch& w,
                                 cudaStream_t s) {
  if (S <= 0) return;
  const int64_t nb = (S + kSortTile - 1) / kSortTile;
  k_gather_keys<<<blocks_of(S, 256), 256, 0, s>>>(key_col, ids, S, w.keys, w.vals);
  uint64_t *kin = w.keys, *kout = w.keys_tmp;
  int32_t *vin = w.vals, *vout = w.vals_tmp;
  for (int shift = 0; shift < 64; shift += 8) {  // 8 passes: the result ends in w.keys / w.vals
    k_radix_hist<<<static_cast<unsigned>(nb), kSortThreads, 0, s>>>(kin, S, shift, w.hist, nb);
    launch_scan_lengths(w.hist, kRadix * nb, w.hist_off, w.scan_tmp, s);
    k_radix_scatter<<<static_cast<unsigned>(nb), kSortThreads, 0, s>>>(kin, vin, S, shift, w.hist_off, nb, kout, vout);
    std::swap(kin, kout);
    std::swap(vin, vout);
  }
  k_group_heads<<<blocks_of(S, 256), 256, 0, s>>>(w.keys, S, w.heads);
  launch_scan_lengths(w.heads, S, w.head_excl, w.scan_tmp, s);
  k_group_starts<<<blocks_of(S, 256), 256, 0, s>>>(w.heads, w.head_excl, S, w.group_start);
  k_pair_counts<<<blocks_of(S, 256), 256, 0, s>>>(w.vals, w.heads, w.head_excl, w.group_start, S, w.counts);
  launch_scan_lengths(w.counts, S, w.pair_off, w.scan_tmp, s);
}

void launch_self_join_pairs_emit(const int32_t* ids, int64_t S, const SelfJoinScratch& w, int32_t* pa, int32_t* pb,
                                 cudaStream_t s) {
  if (S <= 0) return;
  k_emit_pairs<<<blocks_of(S, 256), 256, 0, s>>>(w.vals, w.counts, w.pair_off, ids, S, pa, pb);
}

}  // namespace aiq
