// Token packing of the candidate rows into a variable-length batch.
//
// Every candidate row's prompt is the shared prefix followed by the row's
// tokens (Table 1, AI_IF row: the text column feeds the causal LM; the prompt
// prefix is the instruction shared by all rows); a Q4 pair's prompt is the
// prefix followed by both rows' tokens (Table 2 Q4: AI_IF([A.text, B.text])).
// The prefix is run through the decoder once per query and its keys/values
// are reused by every row
// (causal attention makes the prefix's states independent of what follows),
// so the packed batch holds only each row's own tokens, at positions
// P, P+1, ...  Rows are concatenated with no padding; cu (int64 [S+1]) holds
// each row's start.  The prefill runs over token-budget chunks of
// consecutive rows, the GPU counterpart of the paper's scan over
// micro-batches (Section 3.2): row i belongs to chunk floor(cu[i] / step), so
// a chunk never holds more than step + max_len tokens.
#include "common.cuh"
#include "kernels.h"

namespace aiq {
namespace {

// lens[i] = text length of row ids[i] (plus row ids2[i]'s for a pair prompt);
// pairs += len * P + len * (len + 1) / 2 (the causal query-key pairs its tokens
// attend, for the executed-FLOP count).
__global__ void k_row_lengths(const int64_t* offsets, const int32_t* ids, const int32_t* ids2, int64_t S, int32_t P,
                              int32_t* lens, unsigned long long* pairs) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  unsigned long long pr = 0;
  if (i < S) {
    const int32_t r = ids[i];
    int64_t len = offsets[r + 1] - offsets[r];
    if (ids2) len += offsets[ids2[i] + 1] - offsets[ids2[i]];
    lens[i] = static_cast<int32_t>(len);
    pr = static_cast<unsigned long long>(len * P + len * (len + 1) / 2);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) pr += __shfl_xor_sync(0xffffffffu, pr, o);
  if ((threadIdx.x & 31) == 0 && pr) atomicAdd(pairs, pr);
}

// chunk_rows[2c] = first row i with cu[i] >= c * step (S if none), chunk_rows[2c+1] = cu[that row].
__global__ void k_chunk_bounds(const int64_t* cu, int64_t S, int64_t step, int64_t n_chunks, int64_t* out) {
  const int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (c > n_chunks) return;
  int64_t lo = 0, hi = S;  // lower bound in cu[0..S)
  if (c == n_chunks) {
    lo = S;
  } else {
    const int64_t target = c * step;
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (cu[mid] < target) lo = mid + 1;
      else hi = mid;
    }
  }
  out[2 * c] = lo;
  out[2 * c + 1] = cu[lo];
}

// chunk_rows[2c] = min(c * rows_per_chunk, S), chunk_rows[2c+1] = cu[that row].
__global__ void k_chunk_bounds_rows(const int64_t* cu, int64_t S, int64_t rows_per_chunk, int64_t n_chunks,
                                    int64_t* out) {
  const int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (c > n_chunks) return;
  const int64_t row = c * rows_per_chunk < S ? c * rows_per_chunk : S;
  out[2 * c] = row;
  out[2 * c + 1] = cu[row];
}

// One warp per row: the row's tokens at positions P + j (for a pair prompt the
// first row's text, then the second's); a row with no tokens of its own gets
// last_idx = -1 (its last position is the prefix's last).
__global__ void k_pack_chunk(const int64_t* cu, const int32_t* ids, const int32_t* ids2, const int64_t* offsets,
                             const int32_t* text, int32_t P, int64_t r0, int64_t r1, int32_t* tok, int32_t* pos,
                             int32_t* seq_start, int32_t* last_idx) {
  const int64_t w = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t i = r0 + w;
  if (i >= r1) return;
  const int64_t base = cu[r0];
  const int64_t dst = cu[i] - base;
  const int64_t len = cu[i + 1] - cu[i];
  const int32_t r = ids[i];
  const int32_t* src = text + offsets[r];
  const int64_t len_a = ids2 ? offsets[r + 1] - offsets[r] : len;
  const int64_t off_b = ids2 ? offsets[ids2[i]] : 0;
  for (int64_t j = lane; j < len; j += 32) {
    tok[dst + j] = j < len_a ? src[j] : text[off_b + (j - len_a)];
    pos[dst + j] = static_cast<int32_t>(P + j);
  }
  if (lane == 0) {
    seq_start[w] = static_cast<int32_t>(dst);
    last_idx[w] = len > 0 ? static_cast<int32_t>(dst + len - 1) : -1;
    if (i == r1 - 1) seq_start[w + 1] = static_cast<int32_t>(cu[r1] - base);
  }
}

// Attention work list: one entry per (sequence, block of `tq` query tokens), one block.
__global__ void __launch_bounds__(1024) k_attn_tiles(const int32_t* seq_start, int32_t n, int32_t tq,
                                                     int32_t* tile_seq, int32_t* tile_q0, int32_t* n_tiles) {
  __shared__ int32_t sh[1024];
  int32_t carry = 0;
  for (int32_t b = 0; b < n; b += 1024) {
    const int32_t i = b + threadIdx.x;
    const int32_t cnt = i < n ? (seq_start[i + 1] - seq_start[i] + tq - 1) / tq : 0;
    sh[threadIdx.x] = cnt;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {
      int32_t y = threadIdx.x >= o ? sh[threadIdx.x - o] : 0;
      __syncthreads();
      sh[threadIdx.x] += y;
      __syncthreads();
    }
    int32_t at = carry + sh[threadIdx.x] - cnt;
    for (int32_t q = 0; q < cnt; ++q) {
      tile_seq[at + q] = i;
      tile_q0[at + q] = q * tq;
    }
    carry += sh[1023];
    __syncthreads();
  }
  if (threadIdx.x == 0) *n_tiles = carry;
}

// The prefix as one sequence: tokens, positions 0..P-1, seq_start = {0, P}.
__global__ void k_pack_prefix(const int32_t* prefix, int32_t P, int32_t* tok, int32_t* pos, int32_t* seq_start) {
  for (int j = threadIdx.x; j < P; j += blockDim.x) {
    tok[j] = prefix[j];
    pos[j] = j;
  }
  if (threadIdx.x == 0) {
    seq_start[0] = 0;
    seq_start[1] = P;
  }
}

}  // namespace

void launch_pack_prefix(const int32_t* prefix, int32_t P, int32_t* tok, int32_t* pos, int32_t* seq_start,
                        cudaStream_t s) {
  k_pack_prefix<<<1, 256, 0, s>>>(prefix, P, tok, pos, seq_start);
}

void launch_row_lengths(const int64_t* offsets, const int32_t* ids, int64_t S, int32_t prefix_len, int32_t* lens,
                        unsigned long long* pairs, cudaStream_t s, const int32_t* ids2) {
  if (S <= 0) return;
  k_row_lengths<<<static_cast<unsigned>((S + 255) / 256), 256, 0, s>>>(offsets, ids, ids2, S, prefix_len, lens, pairs);
}

void launch_chunk_bounds(const int64_t* cu, int64_t S, int64_t step, int64_t n_chunks, int64_t* chunk_rows,
                         cudaStream_t s) {
  k_chunk_bounds<<<static_cast<unsigned>((n_chunks + 1 + 127) / 128), 128, 0, s>>>(cu, S, step, n_chunks, chunk_rows);
}

void launch_chunk_bounds_rows(const int64_t* cu, int64_t S, int64_t rows_per_chunk, int64_t n_chunks,
                              int64_t* chunk_rows, cudaStream_t s) {
  k_chunk_bounds_rows<<<static_cast<unsigned>((n_chunks + 1 + 127) / 128), 128, 0, s>>>(cu, S, rows_per_chunk, n_chunks,
                                                                                       chunk_rows);
}

void launch_pack_chunk(const int64_t* cu, const int32_t* ids, const int64_t* offsets, const int32_t* text,
                       int32_t prefix_len, int64_t r0, int64_t r1, int32_t* tok, int32_t* pos, int32_t* seq_start,
                       int32_t* last_idx, cudaStream_t s, const int32_t* ids2) {
  if (r1 <= r0) return;
  const int64_t threads = (r1 - r0) * 32;
  k_pack_chunk<<<static_cast<unsigned>((threads + 255) / 256), 256, 0, s>>>(cu, ids, ids2, offsets, text, prefix_len,
                                                                            r0, r1, tok, pos, seq_start, last_idx);
}

void launch_attn_tiles(const int32_t* seq_start, int32_t n_seqs, int32_t tile_tokens, int32_t* tile_seq,
                       int32_t* tile_q0, int32_t* n_tiles_dev, cudaStream_t s) {
  k_attn_tiles<<<1, 1024, 0, s>>>(seq_start, n_seqs, tile_tokens, tile_seq, tile_q0, n_tiles_dev);
}

}  // namespace aiq
