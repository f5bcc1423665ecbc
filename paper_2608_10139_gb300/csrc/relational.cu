// Relational operators of the unified AI query on the GPU.
//
//  * predicate mask (Table 1, WHERE row): a conjunction of `column op const`
//    terms evaluated over 2048-row tiles, 8 consecutive rows per thread with
//    16-byte vector loads; the result is a bitmask (1 bit per row) plus each
//    tile's survivor count.  A join probe (Section 4: reviews joined with
//    movies on movie id) runs in the same pass for rows that pass the terms.
//  * order-preserving stream compaction: tile counts -> exclusive scan ->
//    each tile re-reads only its 256-byte bitmask slice and writes the ids of
//    its set bits at its offset (reduce-then-scan; no inter-block waits).
//  * open-addressing hash table (int64 key -> build row), linear probing with
//    a bounded probe sequence.
//  * decision (Fig. 2: strict yes > no, or first argmax) and the masked
//    aggregates (Table 1, SELECT row): label counts, yes bitmask for the
//    yes-row ids, GROUP BY build row with warp-aggregated atomics.
#include <cstdio>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace aiq {
namespace {

constexpr int kThreads = 256;  // 256 threads x 8 rows = kRowsPerBlock
constexpr unsigned long long kEmptyKey = 0x8000000000000000ull;

// Raw 8 rows [r0, r0 + 8) of one term's column, as four 16-byte words for
// 4-byte columns (two used) or 64-bit words for int64 columns.
struct TermRows {
  int4 w[4];
};

__device__ __forceinline__ void load_term(const PredDev& p, int64_t r0, int64_t n, TermRows& t) {
  const bool full = r0 + 8 <= n;
  if (p.type == 1) {
    const int64_t* c = static_cast<const int64_t*>(p.col) + r0;
    if (full) {
      const int4* q = reinterpret_cast<const int4*>(c);
#pragma unroll
      for (int j = 0; j < 4; ++j) t.w[j] = __ldg(q + j);
    } else {
      int64_t* v = reinterpret_cast<int64_t*>(t.w);
#pragma unroll
      for (int j = 0; j < 8; ++j) v[j] = r0 + j < n ? c[j] : 0;
    }
  } else {
    const int32_t* c = static_cast<const int32_t*>(p.col) + r0;
    if (full) {
      const int4* q = reinterpret_cast<const int4*>(c);
      t.w[0] = __ldg(q);
      t.w[1] = __ldg(q + 1);
    } else {
      int32_t* v = reinterpret_cast<int32_t*>(t.w);
#pragma unroll
      for (int j = 0; j < 8; ++j) v[j] = r0 + j < n ? c[j] : 0;
    }
  }
}

// The term's 8 result bits for rows loaded by load_term.  The operator is
// resolved once per term (the switch is outside the loop over the 8 values).
template <typename T>
__device__ __forceinline__ uint32_t cmp8(const T* v, int op, T c) {
  uint32_t bits = 0;
  switch (op) {
    case 0:
#pragma unroll
      for (int j = 0; j < 8; ++j) bits |= static_cast<uint32_t>(v[j] < c) << j;
      break;
    case 1:
#pragma unroll
      for (int j = 0; j < 8; ++j) bits |= static_cast<uint32_t>(v[j] <= c) << j;
      break;
    case 2:
#pragma unroll
      for (int j = 0; j < 8; ++j) bits |= static_cast<uint32_t>(v[j] > c) << j;
      break;
    case 3:
#pragma unroll
      for (int j = 0; j < 8; ++j) bits |= static_cast<uint32_t>(v[j] >= c) << j;
      break;
    case 4:
#pragma unroll
      for (int j = 0; j < 8; ++j) bits |= static_cast<uint32_t>(v[j] == c) << j;
      break;
    default:
#pragma unroll
      for (int j = 0; j < 8; ++j) bits |= static_cast<uint32_t>(v[j] != c) << j;
      break;
  }
  return bits;
}

__device__ __forceinline__ uint32_t eval_term(const PredDev& p, const TermRows& t) {
  if (p.type == 1) return cmp8<int64_t>(reinterpret_cast<const int64_t*>(t.w), p.op, p.ivalue);
  if (p.type == 2) return cmp8<float>(reinterpret_cast<const float*>(t.w), p.op, static_cast<float>(p.fvalue));
  // int32: a constant outside the int32 range decides every row alike (as the
  // SQL comparison in int64 would); inside it, compare in 32 bits
  const int32_t* v = reinterpret_cast<const int32_t*>(t.w);
  if (p.ivalue > INT32_MAX || p.ivalue < INT32_MIN) {
    const bool below = p.ivalue > INT32_MAX;  // every value is below the constant
    const bool r = p.op == 0 || p.op == 1 ? below : (p.op == 2 || p.op == 3 ? !below : p.op == 5);
    return r ? 0xFFu : 0u;
  }
  return cmp8<int32_t>(v, p.op, static_cast<int32_t>(p.ivalue));
}

__device__ __forceinline__ int probe_lookup(const ProbeSpec& pr, unsigned long long key) {
  if (key == kEmptyKey) return -1;
  const unsigned long long mask = static_cast<unsigned long long>(pr.capacity - 1);
  unsigned long long slot = hash64(key) & mask;
  for (int64_t i = 0; i < pr.capacity; ++i) {
    const unsigned long long k = pr.table_keys[slot];
    if (k == key) return pr.table_vals[slot];
    if (k == kEmptyKey) return -1;
    slot = (slot + 1) & mask;
  }
  return -1;
}

// Each thread holds one byte of row bits (rows 8*t .. 8*t+7 of the tile);
// assemble 32-bit words (4 lanes each), write them, and return the tile's
// popcount (valid in thread 0).
__device__ __forceinline__ int write_words_and_count(uint32_t byte, uint32_t* bits_tile, int* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t w = byte << (8 * (lane & 3));
  w |= __shfl_xor_sync(0xffffffffu, w, 1);
  w |= __shfl_xor_sync(0xffffffffu, w, 2);
  if ((lane & 3) == 0) bits_tile[threadIdx.x >> 2] = w;
  int c = __popc(byte);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if (lane == 0) red[warp] = c;
  __syncthreads();
  int total = 0;
  if (threadIdx.x == 0)
    for (int i = 0; i < kThreads / 32; ++i) total += red[i];
  return total;
}

// Evaluates the terms (and the join probe) on one 2048-row tile; thread t
// covers rows 8t .. 8t+7.  `stage` holds the tile's column chunks when the
// tile is full; the ragged last tile reads global memory directly.
__device__ __forceinline__ void predicate_tile(const PredSet& ps, const ProbeSpec& probe, int64_t n, int64_t tile,
                                               const uint8_t* stage, const int* s_off, uint32_t* bits,
                                               int32_t* block_counts, int* red) {
  const int64_t r0 = tile * kRowsPerBlock + threadIdx.x * 8;
  uint32_t byte = 0;
  if (r0 < n) {
    byte = r0 + 8 <= n ? 0xFFu : ((1u << (n - r0)) - 1u);
    for (int i = 0; i < ps.n; ++i) {
      TermRows t;
      if (stage) {
        const int4* src = reinterpret_cast<const int4*>(stage + s_off[i]) + threadIdx.x * (ps.p[i].type == 1 ? 4 : 2);
        t.w[0] = src[0];
        t.w[1] = src[1];
        if (ps.p[i].type == 1) {
          t.w[2] = src[2];
          t.w[3] = src[3];
        }
      } else {
        load_term(ps.p[i], r0, n, t);
      }
      byte &= eval_term(ps.p[i], t);
    }
    if (probe.keys) {
#pragma unroll 1
      for (int j = 0; j < 8; ++j) {
        if (byte & (1u << j)) {
          const int m = probe_lookup(probe, static_cast<unsigned long long>(probe.keys[r0 + j]));
          if (m < 0) byte &= ~(1u << j);
          else probe.match_out[r0 + j] = m;
        }
      }
    }
  }
  const int total = write_words_and_count(byte, bits + tile * (kRowsPerBlock / 32), red);
  if (threadIdx.x == 0) block_counts[tile] = total;
}

// One 2048-row tile per block.  Thread 0 first asks the bulk-copy engine to
// pull every term's column chunk of the tile (2048 x 4 or 8 bytes) into L2,
// so all columns stream from DRAM at once while each thread's own 16-byte
// loads of successive terms follow one after the other.
__global__ void __launch_bounds__(kThreads) k_predicate_mask(PredSet ps, ProbeSpec probe, int64_t n, uint32_t* bits,
                                                             int32_t* block_counts, int* err) {
  __shared__ int red[kThreads / 32];
  const int64_t tile = blockIdx.x;
  if (threadIdx.x == 0 && (tile + 1) * kRowsPerBlock <= n) {
    for (int i = 1; i < ps.n; ++i) {
      const int esz = ps.p[i].type == 1 ? 8 : 4;
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const uint8_t*>(ps.p[i].col) +
                                                                        tile * kRowsPerBlock * esz),
                   "r"(kRowsPerBlock * esz)
                   : "memory");
    }
  }
  predicate_tile(ps, probe, n, tile, nullptr, nullptr, bits, block_counts, red);
  (void)err;
}

// The common case, 1..4 terms on 4-byte columns and no join probe: every
// term's loads are issued before the first compare, in a coalesced layout
// (lane l of warp w takes rows 4l..4l+3 and 128+4l..128+4l+3 of the warp's
// 256 rows, so one 16-byte load instruction covers 512 contiguous bytes),
// and eight lanes' nibbles form one bitmask word.  Same bitmask and tile
// counts as k_predicate_mask.
template <int NT>
__global__ void __launch_bounds__(kThreads) k_predicate_mask4(PredSet ps, int64_t n, uint32_t* bits,
                                                              int32_t* block_counts) {
  __shared__ int red[kThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t ra = static_cast<int64_t>(blockIdx.x) * kRowsPerBlock + warp * 256 + lane * 4;
  const int64_t rb = ra + 128;
  int4 va[NT], vb[NT];
  const bool full = rb + 4 <= n;
#pragma unroll
  for (int i = 0; i < NT; ++i) {
    const int32_t* c = static_cast<const int32_t*>(ps.p[i].col);
    if (full) {
      va[i] = __ldg(reinterpret_cast<const int4*>(c + ra));
      vb[i] = __ldg(reinterpret_cast<const int4*>(c + rb));
    } else {
      int32_t* x = reinterpret_cast<int32_t*>(&va[i]);
      int32_t* y = reinterpret_cast<int32_t*>(&vb[i]);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        x[j] = ra + j < n ? c[ra + j] : 0;
        y[j] = rb + j < n ? c[rb + j] : 0;
      }
    }
  }
  uint32_t byte = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) byte |= (static_cast<uint32_t>(ra + j < n) << j) | (static_cast<uint32_t>(rb + j < n) << (4 + j));
#pragma unroll
  for (int i = 0; i < NT; ++i) {
    TermRows t;
    t.w[0] = va[i];
    t.w[1] = vb[i];
    // eval_term's value j < 4 is row ra + j, value 4 + j is row rb + j
    byte &= eval_term(ps.p[i], t);
  }
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    uint32_t w = ((byte >> (4 * h)) & 0xFu) << (4 * (lane & 7));
    w |= __shfl_xor_sync(0xffffffffu, w, 1);
    w |= __shfl_xor_sync(0xffffffffu, w, 2);
    w |= __shfl_xor_sync(0xffffffffu, w, 4);
    if ((lane & 7) == 0) bits[blockIdx.x * int64_t(kRowsPerBlock / 32) + warp * 8 + h * 4 + (lane >> 3)] = w;
  }
  int c = __popc(byte);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if (lane == 0) red[warp] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    int total = 0;
    for (int i = 0; i < kThreads / 32; ++i) total += red[i];
    block_counts[blockIdx.x] = total;
  }
}

// Block-wide exclusive scan of one int per thread (kThreads threads).
__device__ __forceinline__ int block_excl_scan(int v, int* sh, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int s = lane < kThreads / 32 ? sh[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    if (lane < kThreads / 32) sh[lane] = s;
  }
  __syncthreads();
  const int before = warp ? sh[warp - 1] : 0;
  *total = sh[kThreads / 32 - 1];
  return before + x - v;
}

constexpr int kCompactWarps = 4;  // warps (= 2048-row tiles at a time) per compaction block

// One warp per 2048-row tile: lane l owns bitmask words l and 32 + l of the
// tile (two coalesced loads).  In two passes (words 0..31, then 32..63) a warp
// shuffle scan gives every lane its output position and the lane writes the
// row offsets of its word's set bits, in order, into the warp's own 16-bit
// shared-memory slice; the slice is then written out as one coalesced run of
// ids.  No block-wide barrier is involved.  A payload (the join's build row
// per probe row) is gathered straight to its output position (PAYLOAD).
template <bool PAYLOAD>
__global__ void __launch_bounds__(kCompactWarps * 32) k_compact(const uint32_t* bits, const int64_t* block_offsets,
                                                                int64_t n, int32_t* ids, const int32_t* payload,
                                                                int32_t* payload_out) {
  __shared__ uint16_t s_ids[kCompactWarps][kRowsPerBlock];  // row offsets within the tile
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t n_tiles = (n + kRowsPerBlock - 1) / kRowsPerBlock;
  const int64_t tile = static_cast<int64_t>(blockIdx.x) * kCompactWarps + warp;
  if (tile < n_tiles) {
    const uint32_t* wt = bits + tile * (kRowsPerBlock / 32);
    const uint32_t wa = wt[lane], wb = wt[32 + lane];
    const int64_t out = block_offsets[tile];
    const int64_t tile0 = tile * kRowsPerBlock;
    int at0 = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      uint32_t b = h ? wb : wa;
      const int c = __popc(b);
      int incl = c;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      int at = at0 + incl - c;
      const int base = (h * 32 + lane) * 32;
      while (b) {
        const int j = __ffs(b) - 1;
        b &= b - 1;
        s_ids[warp][at] = static_cast<uint16_t>(base + j);
        if (PAYLOAD) payload_out[out + at] = payload[tile0 + base + j];  // joins: a gather, written in place
        ++at;
      }
      at0 += __shfl_sync(0xffffffffu, incl, 31);
    }
    __syncwarp();
    for (int i = lane; i < at0; i += 32) ids[out + i] = static_cast<int32_t>(tile0 + s_ids[warp][i]);
  }
}

// ---------------------------------------------------------------- scans ---
// Tile sums (2048 ints per block) -> single-block scan of the tile sums ->
// per-tile scan with the tile's offset.

__global__ void __launch_bounds__(kThreads) k_tile_sums(const int32_t* in, int64_t n, int64_t* sums) {
  __shared__ int64_t red[kThreads / 32];
  const int64_t base = static_cast<int64_t>(blockIdx.x) * kRowsPerBlock;
  int64_t s = 0;
  for (int i = threadIdx.x; i < kRowsPerBlock; i += kThreads)
    if (base + i < n) s += in[base + i];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    int64_t t = 0;
    for (int i = 0; i < kThreads / 32; ++i) t += red[i];
    sums[blockIdx.x] = t;
  }
}

// Exclusive scan of n int64 (or int32) values into out[0..n], one block of 1024
// threads, each scanning a contiguous run sequentially.
template <typename T>
__global__ void __launch_bounds__(1024) k_scan_single(const T* in, int64_t n, int64_t* out) {
  __shared__ int64_t sh[1024];
  const int64_t per = (n + 1023) / 1024;
  const int64_t b = threadIdx.x * per;
  int64_t s = 0;
  for (int64_t i = b; i < b + per && i < n; ++i) s += in[i];
  sh[threadIdx.x] = s;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {
    int64_t y = threadIdx.x >= o ? sh[threadIdx.x - o] : 0;
    __syncthreads();
    sh[threadIdx.x] += y;
    __syncthreads();
  }
  int64_t run = sh[threadIdx.x] - s;
  for (int64_t i = b; i < b + per && i < n; ++i) {
    out[i] = run;
    run += in[i];
  }
  if (threadIdx.x == 1023) out[n] = sh[1023];
}

__global__ void __launch_bounds__(kThreads) k_tile_scan(const int32_t* in, int64_t n, const int64_t* tile_off,
                                                        int64_t* out) {
  __shared__ int sh[kThreads / 32];
  const int64_t base = static_cast<int64_t>(blockIdx.x) * kRowsPerBlock + threadIdx.x * 8;
  int v[8];
  int s = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    v[j] = base + j < n ? in[base + j] : 0;
    s += v[j];
  }
  int total;
  int pre = block_excl_scan(s, sh, &total);
  int64_t run = tile_off[blockIdx.x] + pre;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    if (base + j < n) out[base + j] = run;
    run += v[j];
  }
  if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) out[n] = tile_off[gridDim.x];
}

// ----------------------------------------------------------- hash build ---

__global__ void k_hash_build(const int64_t* keys, const int32_t* rows, int64_t n, unsigned long long* tk,
                             int32_t* tv, int64_t cap, int* err) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const int32_t row = rows[i];
  const unsigned long long key = static_cast<unsigned long long>(keys[row]);
  if (key == kEmptyKey) {
    set_dev_error(err, DEVERR_SENTINEL_KEY);
    return;
  }
  const unsigned long long mask = static_cast<unsigned long long>(cap - 1);
  unsigned long long slot = hash64(key) & mask;
  for (int64_t step = 0; step < cap; ++step) {
    const unsigned long long prev = atomicCAS(tk + slot, kEmptyKey, key);
    if (prev == kEmptyKey) {
      tv[slot] = row;
      return;
    }
    if (prev == key) {
      set_dev_error(err, DEVERR_DUP_BUILD_KEY);
      return;
    }
    slot = (slot + 1) & mask;
  }
  set_dev_error(err, DEVERR_HASH_FULL);
}

__global__ void k_fill_u64(unsigned long long* p, int64_t n, unsigned long long v) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    p[i] = v;
}

// ------------------------------------------------------ decide/aggregate ---

__global__ void __launch_bounds__(kThreads) k_decide(const float* logits, int64_t S, int K, int32_t* decision,
                                                     uint32_t* yes_bits, int32_t* block_counts,
                                                     unsigned long long* label_counts) {
  __shared__ int red[kThreads / 32];
  __shared__ unsigned int hist[16];
  if (threadIdx.x < 16) hist[threadIdx.x] = 0;
  __syncthreads();
  const int64_t r0 = static_cast<int64_t>(blockIdx.x) * kRowsPerBlock + threadIdx.x * 8;
  uint32_t byte = 0;
  for (int j = 0; j < 8; ++j) {
    const int64_t r = r0 + j;
    if (r >= S) break;
    const float* z = logits + r * K;
    int d;
    if (K == 2) {
      d = z[0] > z[1] ? 1 : 0;  // strict: a tie is "no"
      byte |= static_cast<uint32_t>(d) << j;
      atomicAdd(&hist[d ? 0 : 1], 1u);
    } else {
      d = 0;
      float best = z[0];
      for (int k = 1; k < K; ++k)
        if (z[k] > best) {
          best = z[k];
          d = k;
        }
      atomicAdd(&hist[d], 1u);
    }
    decision[r] = d;
  }
  const int total = write_words_and_count(byte, yes_bits + static_cast<int64_t>(blockIdx.x) * (kRowsPerBlock / 32), red);
  if (threadIdx.x == 0) block_counts[blockIdx.x] = total;
  if (threadIdx.x < K && hist[threadIdx.x]) atomicAdd(label_counts + threadIdx.x, (unsigned long long)hist[threadIdx.x]);
}

__global__ void __launch_bounds__(kThreads) k_flag_mask(const int32_t* flags, int64_t n, uint32_t* bits,
                                                         int32_t* block_counts) {
  __shared__ int red[kThreads / 32];
  const int64_t r0 = static_cast<int64_t>(blockIdx.x) * kRowsPerBlock + threadIdx.x * 8;
  uint32_t byte = 0;
  for (int j = 0; j < 8 && r0 + j < n; ++j) byte |= static_cast<uint32_t>(flags[r0 + j] != 0) << j;
  const int total = write_words_and_count(byte, bits + static_cast<int64_t>(blockIdx.x) * (kRowsPerBlock / 32), red);
  if (threadIdx.x == 0) block_counts[blockIdx.x] = total;
}

// Fixed-order reductions (warp shuffle tree, then the warps in order) so that
// the float sum is the same on every run.
template <typename T>
__device__ __forceinline__ T block_sum_fixed(T v, T* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  T t = 0;
  if (threadIdx.x == 0)
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) t += sh[w];
  return t;
}

template <typename T, typename C>
__global__ void __launch_bounds__(kThreads) k_masked_sum(const int32_t* decision, const int32_t* ids, const C* col,
                                                         int64_t S, T* partial) {
  __shared__ T sh[kThreads / 32];
  const int64_t r0 = static_cast<int64_t>(blockIdx.x) * kRowsPerBlock + threadIdx.x * 8;
  T acc = 0;
  for (int j = 0; j < 8; ++j) {
    const int64_t i = r0 + j;
    if (i < S && decision[i] == 1) acc += static_cast<T>(col[ids[i]]);
  }
  const T t = block_sum_fixed<T>(acc, sh);
  if (threadIdx.x == 0) partial[blockIdx.x] = t;
}

template <typename T>
__global__ void __launch_bounds__(1024) k_sum_final(const T* partial, int64_t n, T* out) {
  __shared__ T sh[32];
  T acc = 0;
  for (int64_t i = threadIdx.x; i < n; i += 1024) acc += partial[i];
  const T t = block_sum_fixed<T>(acc, sh);
  if (threadIdx.x == 0) *out = t;
}

__global__ void k_group_build(const int32_t* decision, const int32_t* build_rows, int64_t S,
                              unsigned long long* counts) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  const bool yes = i < S && decision[i] == 1;
  const unsigned active = __ballot_sync(0xffffffffu, yes);
  if (!yes) return;
  const int key = build_rows[i];
  // lanes of the warp that hit the same group add once (skewed foreign keys)
  const unsigned same = __match_any_sync(active, key);
  if ((threadIdx.x & 31) == __ffs(same) - 1) atomicAdd(counts + key, (unsigned long long)__popc(same));
}

__global__ void __launch_bounds__(kThreads) k_nonzero_mask(const unsigned long long* counts, int64_t n, uint32_t* bits,
                                                           int32_t* block_counts) {
  __shared__ int red[kThreads / 32];
  const int64_t r0 = static_cast<int64_t>(blockIdx.x) * kRowsPerBlock + threadIdx.x * 8;
  uint32_t byte = 0;
  for (int j = 0; j < 8; ++j)
    if (r0 + j < n && counts[r0 + j] != 0) byte |= 1u << j;
  const int total = write_words_and_count(byte, bits + static_cast<int64_t>(blockIdx.x) * (kRowsPerBlock / 32), red);
  if (threadIdx.x == 0) block_counts[blockIdx.x] = total;
}

__global__ void k_gather_groups(const int32_t* rows, int64_t g, const int64_t* keys, const unsigned long long* counts,
                                int64_t* keys_out, int64_t* counts_out) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= g) return;
  const int32_t r = rows[i];
  keys_out[i] = keys[r];
  counts_out[i] = static_cast<int64_t>(counts[r]);
}

inline unsigned blocks_for(int64_t n, int64_t per) { return static_cast<unsigned>((n + per - 1) / per); }

}  // namespace

void launch_predicate_mask(const PredSet& ps, const ProbeSpec& probe, int64_t n_rows, uint32_t* bits,
                           int32_t* block_counts, int* err, cudaStream_t s) {
  if (n_rows <= 0) return;
  const unsigned grid = blocks_for(n_rows, kRowsPerBlock);
  bool four = ps.n >= 1 && ps.n <= 4 && !probe.keys;
  for (int i = 0; i < ps.n; ++i)
    four = four && ps.p[i].type != 1 && (reinterpret_cast<uintptr_t>(ps.p[i].col) & 15) == 0;
  if (four) {
    switch (ps.n) {
      case 1: k_predicate_mask4<1><<<grid, kThreads, 0, s>>>(ps, n_rows, bits, block_counts); break;
      case 2: k_predicate_mask4<2><<<grid, kThreads, 0, s>>>(ps, n_rows, bits, block_counts); break;
      case 3: k_predicate_mask4<3><<<grid, kThreads, 0, s>>>(ps, n_rows, bits, block_counts); break;
      default: k_predicate_mask4<4><<<grid, kThreads, 0, s>>>(ps, n_rows, bits, block_counts); break;
    }
  } else {
    k_predicate_mask<<<grid, kThreads, 0, s>>>(ps, probe, n_rows, bits, block_counts, err);
  }
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    char buf[160];
    snprintf(buf, sizeof(buf), "predicate mask launch (grid %u, terms %d)", grid, ps.n);
    set_launch_error(buf, e);
  }
}

void launch_scan_counts(const int32_t* counts, int64_t n, int64_t* offsets, cudaStream_t s) {
  k_scan_single<int32_t><<<1, 1024, 0, s>>>(counts, n, offsets);
}

void launch_compact(const uint32_t* bits, const int64_t* block_offsets, int64_t n_rows, int32_t* ids_out,
                    const int32_t* payload, int32_t* payload_out, cudaStream_t s) {
  if (n_rows <= 0) return;
  const unsigned grid = blocks_for(n_rows, int64_t(kRowsPerBlock) * kCompactWarps);  // one tile per warp
  if (payload_out)
    k_compact<true><<<grid, kCompactWarps * 32, 0, s>>>(bits, block_offsets, n_rows, ids_out, payload, payload_out);
  else
    k_compact<false><<<grid, kCompactWarps * 32, 0, s>>>(bits, block_offsets, n_rows, ids_out, payload, payload_out);
}

void launch_hash_build(const int64_t* keys, const int32_t* rows, int64_t n, unsigned long long* table_keys,
                       int32_t* table_vals, int64_t capacity, int* err, cudaStream_t s) {
  if (n <= 0) return;
  k_hash_build<<<blocks_for(n, 256), 256, 0, s>>>(keys, rows, n, table_keys, table_vals, capacity, err);
}

void launch_fill_u64(unsigned long long* p, int64_t n, unsigned long long v, cudaStream_t s) {
  if (n <= 0) return;
  const unsigned g = blocks_for(n, 256) < 4096 ? blocks_for(n, 256) : 4096;
  k_fill_u64<<<g, 256, 0, s>>>(p, n, v);
}

void launch_scan_lengths(const int32_t* lens, int64_t S, int64_t* cu, int64_t* scratch_blocks, cudaStream_t s) {
  // scratch_blocks: >= 2 * (tiles + 1) int64
  const int64_t tiles = (S + kRowsPerBlock - 1) / kRowsPerBlock;
  if (tiles == 0) {
    cudaMemsetAsync(cu, 0, sizeof(int64_t), s);
    return;
  }
  int64_t* sums = scratch_blocks;
  int64_t* off = scratch_blocks + tiles + 1;
  k_tile_sums<<<static_cast<unsigned>(tiles), kThreads, 0, s>>>(lens, S, sums);
  k_scan_single<int64_t><<<1, 1024, 0, s>>>(sums, tiles, off);
  k_tile_scan<<<static_cast<unsigned>(tiles), kThreads, 0, s>>>(lens, S, off, cu);
}

void launch_decide(const float* logits, int64_t S, int K, int32_t* decision, uint32_t* yes_bits,
                   int32_t* block_counts, unsigned long long* label_counts, cudaStream_t s) {
  if (S <= 0) return;
  k_decide<<<blocks_for(S, kRowsPerBlock), kThreads, 0, s>>>(logits, S, K, decision, yes_bits, block_counts,
                                                             label_counts);
}

void launch_flag_mask(const int32_t* flags, int64_t n, uint32_t* bits, int32_t* block_counts, cudaStream_t s) {
  if (n <= 0) return;
  k_flag_mask<<<blocks_for(n, kRowsPerBlock), kThreads, 0, s>>>(flags, n, bits, block_counts);
}

void launch_masked_sum(const int32_t* decision, const int32_t* ids, const void* col, int type, int64_t S,
                       void* partial, void* out, cudaStream_t s) {
  const unsigned nb = S > 0 ? blocks_for(S, kRowsPerBlock) : 0;
  if (type == 2) {
    if (nb) k_masked_sum<double, float><<<nb, kThreads, 0, s>>>(decision, ids, static_cast<const float*>(col), S,
                                                                 static_cast<double*>(partial));
    k_sum_final<double><<<1, 1024, 0, s>>>(static_cast<const double*>(partial), nb, static_cast<double*>(out));
  } else {
    // integers sum modulo 2^64 (unsigned arithmetic: a wrap is defined), read back as int64
    unsigned long long* pp = static_cast<unsigned long long*>(partial);
    if (nb && type == 0)
      k_masked_sum<unsigned long long, int32_t><<<nb, kThreads, 0, s>>>(decision, ids,
                                                                         static_cast<const int32_t*>(col), S, pp);
    if (nb && type == 1)
      k_masked_sum<unsigned long long, long long><<<nb, kThreads, 0, s>>>(decision, ids,
                                                                           static_cast<const long long*>(col), S, pp);
    k_sum_final<unsigned long long><<<1, 1024, 0, s>>>(pp, nb, static_cast<unsigned long long*>(out));
  }
}

void launch_group_build(const int32_t* decision, const int32_t* cand_build_rows, int64_t S,
                        unsigned long long* group_counts, cudaStream_t s) {
  if (S <= 0) return;
  k_group_build<<<blocks_for(S, 256), 256, 0, s>>>(decision, cand_build_rows, S, group_counts);
}

void launch_nonzero_mask(const unsigned long long* counts, int64_t n, uint32_t* bits, int32_t* block_counts,
                         cudaStream_t s) {
  if (n <= 0) return;
  k_nonzero_mask<<<blocks_for(n, kRowsPerBlock), kThreads, 0, s>>>(counts, n, bits, block_counts);
}

void launch_gather_groups(const int32_t* rows, int64_t g, const int64_t* build_keys,
                          const unsigned long long* counts, int64_t* keys_out, int64_t* counts_out,
                          cudaStream_t s) {
  if (g <= 0) return;
  k_gather_groups<<<blocks_for(g, 256), 256, 0, s>>>(rows, g, build_keys, counts, keys_out, counts_out);
}

}  // namespace aiq
