// Internal host-side launchers of the library's CUDA kernels.  The C-ABI
// layer (aiq_api.cu) is the only caller; none of this is exported.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace aiq {

// ------------------------------------------------------------------ GEMM ---
enum GemmEpi : int {
  EPI_F16 = 0,        // out fp16 [M, N] = acc
  EPI_ROPE_F16 = 1,   // as EPI_F16, rotary embedding applied to columns < rope_cols
  EPI_RESID_F32 = 2,  // out fp32 [M, N] += acc  (residual stream update)
  EPI_SWIGLU_F16 = 3, // B interleaves gate/up blocks of BN/2 rows: out fp16 [M, N/2] = silu(g) * u
  EPI_ARGMAX = 4,     // per row: max over columns of acc + bias[col] and its first column, folded into
                      // best[row] with a 64-bit atomicMax of (order-preserving value bits, ~col)
  EPI_RESID_ADD = 5,  // out fp32 [M, N] += acc by TMA reduce-add tiles (no xh_out / ss_out)
};

struct GemmEpilogue {
  int kind = EPI_F16;
  void* out = nullptr;
  int64_t ldo = 0;                     // elements
  const int32_t* positions = nullptr;  // ROPE: per-row position
  const float* rope_cos = nullptr;     // ROPE: [max_pos, head_dim/2]
  const float* rope_sin = nullptr;
  int rope_cols = 0;
  int head_dim = 0;
  int* err = nullptr;
  // RMSNorm fused across GEMMs:
  //  - consumer (ROPE / SWIGLU): scale each accumulator row by
  //    rsqrt(sum(row_ss[row][0..ss_parts)) / d_norm + eps) before the epilogue;
  //  - producer (RESID): also write the new residual as fp16 (xh_out), times
  //    the next norm's gain (xh_gain, bf16 [N]) when given, and the unscaled
  //    residual's per-128-column sums of squares (ss_out [row][n / 128]).
  const float* row_ss = nullptr;
  int ss_parts = 0;
  float d_norm = 1.f;
  float eps = 0.f;
  __half* xh_out = nullptr;
  const uint16_t* xh_gain = nullptr;
  float* ss_out = nullptr;
  // SWIGLU: when > 0, also write fp16(v - fp16(v)) lo_off elements after each
  // output (a two-term operand for the next, K-doubled, GEMM)
  int64_t lo_off = 0;
  // EPI_ARGMAX: fp32 bias [N] (-inf marks padding columns) and the per-row packed result
  const float* bias = nullptr;
  unsigned long long* best = nullptr;
};

// C = A[M,K] * B[N,K]^T with fp16 operands and fp32 accumulation on tcgen05.
// Requires K % 64 == 0, N % bn == 0, bn in {128, 256}, 16-byte aligned rows.
// pair: 256 x 256 tiles on clusters of two CTAs (cta_group::2); needs bn == 256.
// Returns 0 or a cudaError_t value.
int gemm_f16_tcgen05(const __half* A, int64_t lda, const __half* B, int64_t ldb, int M, int N, int K, int bn,
                     bool pair, const GemmEpilogue& ep, int num_sms, cudaStream_t stream);

// ------------------------------------------------------------ relational ---
struct PredDev {
  const void* col;
  int32_t type;   // 0 int32, 1 int64, 2 float32
  int32_t op;     // aiq_cmp
  int64_t ivalue;
  double fvalue;
};
constexpr int kMaxPreds = 8;
struct PredSet {
  PredDev p[kMaxPreds];
  int n;
};

constexpr int kRowsPerBlock = 2048;  // rows per predicate / compaction block (64 bitmask words)

// Hash-join probe evaluated together with the probe-side predicate.
struct ProbeSpec {
  const int64_t* keys = nullptr;  // probe key column (nullptr: no join)
  const unsigned long long* table_keys = nullptr;
  const int32_t* table_vals = nullptr;
  int64_t capacity = 0;           // power of two
  int32_t* match_out = nullptr;   // build row per probe row (valid where the bit is set)
};

// mask bits + per-block survivor counts.
void launch_predicate_mask(const PredSet& ps, const ProbeSpec& probe, int64_t n_rows, uint32_t* bits,
                           int32_t* block_counts, int* err, cudaStream_t s);
// Exclusive scan of n int32 counts into int64 offsets[n+1] (one block).
void launch_scan_counts(const int32_t* counts, int64_t n, int64_t* offsets, cudaStream_t s);
// Order-preserving compaction of set bits: ids_out[k] = row of the k-th set bit;
// optionally gathers `payload[row]` into payload_out[k].
void launch_compact(const uint32_t* bits, const int64_t* block_offsets, int64_t n_rows, int32_t* ids_out,
                    const int32_t* payload, int32_t* payload_out, cudaStream_t s);

void launch_hash_build(const int64_t* keys, const int32_t* rows, int64_t n, unsigned long long* table_keys,
                       int32_t* table_vals, int64_t capacity, int* err, cudaStream_t s);
void launch_fill_u64(unsigned long long* p, int64_t n, unsigned long long v, cudaStream_t s);

// ------------------------------------------------------------------ pack ---
// lens[i] = text length of row ids[i]; *pairs += causal (q, k) pairs of its tokens
// (prefix keys included).
// ids2 (optional): a second row per sequence whose text follows the first's (Q4 pairs).
void launch_row_lengths(const int64_t* offsets, const int32_t* ids, int64_t S, int32_t prefix_len, int32_t* lens,
                        unsigned long long* pairs, cudaStream_t s, const int32_t* ids2 = nullptr);
// Exclusive scan of int32 lengths into int64 cu[S+1] (multi-block).
void launch_scan_lengths(const int32_t* lens, int64_t S, int64_t* cu, int64_t* scratch_blocks, cudaStream_t s);
// chunk_rows[c] = first row whose start offset >= c * budget_step, c = 0..n_chunks.
void launch_chunk_bounds(const int64_t* cu, int64_t S, int64_t step, int64_t n_chunks, int64_t* chunk_rows,
                         cudaStream_t s);
// Chunks of equal row counts: chunk_rows[2c] = min(c * rows_per_chunk, S), [2c+1] = cu[that row].
void launch_chunk_bounds_rows(const int64_t* cu, int64_t S, int64_t rows_per_chunk, int64_t n_chunks,
                              int64_t* chunk_rows, cudaStream_t s);
// Pack rows [r0, r1) of a chunk: their own tokens at positions prefix_len + j,
// chunk-local sequence starts and last-token index (-1 for a row without tokens).
void launch_pack_chunk(const int64_t* cu, const int32_t* ids, const int64_t* offsets, const int32_t* text,
                       int32_t prefix_len, int64_t r0, int64_t r1, int32_t* tok, int32_t* pos, int32_t* seq_start,
                       int32_t* last_idx, cudaStream_t s, const int32_t* ids2 = nullptr);
// The shared prefix as a single sequence at positions 0..P-1.
void launch_pack_prefix(const int32_t* prefix, int32_t P, int32_t* tok, int32_t* pos, int32_t* seq_start,
                        cudaStream_t s);
// Attention work list of a chunk: one entry per (sequence, block of tile_tokens query tokens).
void launch_attn_tiles(const int32_t* seq_start, int32_t n_seqs, int32_t tile_tokens, int32_t* tile_seq,
                       int32_t* tile_q0, int32_t* n_tiles_dev, cudaStream_t s);

// --------------------------------------------------------------- prefill ---
// dst[r * ldd + c] = fp16(src[r][c]) (exact for bf16 values in fp16's range;
// rows optionally interleaved in blocks, see k_bf16_to_f16; ldd 0 = cols).
void launch_bf16_to_f16(const uint16_t* src, __half* dst, int64_t rows, int64_t cols, int interleave_block,
                        int64_t half_rows, int* err, cudaStream_t s, int64_t ldd = 0);
void launch_rope_table(float* cos_t, float* sin_t, int max_pos, int head_dim, float theta, cudaStream_t s);
// Embedding rows into the fp32 residual; with xh/ss also its fp16 copy (times
// `gain`, the first layer's attention-norm gain, when given) and the unscaled
// row's per-128-column sums of squares (the first layer's fused RMSNorm input).
void launch_embed(const int32_t* tok, int64_t T, const uint16_t* emb, int d, float* resid, __half* xh, float* ss,
                  const uint16_t* gain, int* err, cudaStream_t s);
// g may be null (unit gain).  split: out rows are 2d wide, fp16(v) then
// fp16(v - fp16(v)) (a two-term operand for a K-doubled GEMM).
void launch_rmsnorm(const float* x, int64_t T, int d, const uint16_t* g, float eps, __half* out, int* err,
                    cudaStream_t s, bool split = false);
// prefix_kv (optional): [P, 2 Hkv hd] fp16 keys then values of a shared prefix that
// every sequence's queries also attend (prefix positions precede the sequence).
void launch_attention(const __half* qkv, int64_t T, const int32_t* seq_start, const int32_t* tile_seq,
                      const int32_t* tile_q0, int n_tiles_max, const int32_t* n_tiles_dev, int Hq, int Hkv,
                      int hd, const __half* prefix_kv, int P, __half* out, int* err, cudaStream_t s);
// Gathers each row's last-token attention output and residual into dense [n, .]
// buffers for the final layer's row-only O-projection and MLP.
void launch_gather_last(const __half* att, int ld_att, const float* resid, int d, const int32_t* last_idx, int64_t n,
                        __half* att_out, float* resid_out, int32_t* last_compact, cudaStream_t s);
// tcgen05 attention (head_dim 64 or 128, query heads per KV head dividing 128):
// work items of tile_tokens = 128 / (Hq / Hkv) tokens x one KV-head group.
bool attention_tc_supported(int hd, int Hq, int Hkv);
int attention_tc_tile_tokens(int Hq, int Hkv);
int launch_attention_tc(const __half* qkv, int64_t T, const int32_t* seq_start, const int32_t* tile_seq,
                        const int32_t* tile_q0, int n_tiles_max, const int32_t* n_tiles_dev, int Hq, int Hkv, int hd,
                        const __half* prefix_kv, int P, __half* out, int* err, int num_sms, cudaStream_t s);
// last_idx[r] < 0 reads prefix_last (fp32 [d]) instead of a row of resid.
void launch_label_head(const float* resid, const int32_t* last_idx, const float* prefix_last, int64_t n_rows, int d,
                       const uint16_t* g, float eps, const uint16_t* lm_head, const uint16_t* lm_bias,
                       const int32_t* labels, int n_labels, float* logits_out, cudaStream_t s);

// ------------------------------------------------------------- aggregate ---
// decision per row from logits [S, K] (K == 2: strict yes > no; K > 2: first argmax),
// yes-bitmask (K == 2), per-block yes counts, label counts [K] (int64, atomics).
void launch_decide(const float* logits, int64_t S, int K, int32_t* decision, uint32_t* yes_bits,
                   int32_t* block_counts, unsigned long long* label_counts, cudaStream_t s);
// Fig. 2's masked reduction: SUM(col[ids[i]]) over rows with decision[i] == 1,
// deterministic (fixed-order block and final reductions).  type: 0 int32,
// 1 int64 (exact int64 sum), 2 float32 (fp64 sum).  partial: >= ceil(S / 2048)
// 8-byte slots; out: one 8-byte slot (int64 or double by type).
void launch_masked_sum(const int32_t* decision, const int32_t* ids, const void* col, int type, int64_t S,
                       void* partial, void* out, cudaStream_t s);
// group counts[build_row] += 1 for yes rows.
void launch_group_build(const int32_t* decision, const int32_t* cand_build_rows, int64_t S,
                        unsigned long long* group_counts, cudaStream_t s);
// bits of non-zero group counts + per-block counts.
void launch_nonzero_mask(const unsigned long long* counts, int64_t n, uint32_t* bits, int32_t* block_counts,
                         cudaStream_t s);
void launch_gather_groups(const int32_t* rows, int64_t g, const int64_t* build_keys,
                          const unsigned long long* counts, int64_t* keys_out, int64_t* counts_out,
                          cudaStream_t s);

// ------------------------------------------------------------- self-test ---
// One CTA of two warps waiting on an mbarrier phase that never completes (warp 0
// with limit_ns, warp 1 with 4 x limit_ns; see aiq_op_wait_expiry_selftest).
int launch_wait_expiry(uint64_t limit_ns, int* err, cudaStream_t s);

// ---------------------------------------------------------------- decode ---
// Decode attention of R single-token rows (row r's token: q/k/v in qkv row r).
// Keys of row r: the P shared-prefix rows of pkv, its own prompt rows
// kvc[seq_start[r] .. seq_start[r+1]), then its generated slots gkv[r][0 .. slot]
// (this step's key/value are first written to slot `slot`).  Layouts [.][2 Hkv hd]
// (keys then values).  Returns 0 or a cudaError_t value.
int launch_decode_attention(const __half* qkv, int64_t ldq, int R, int Hq, int Hkv, int hd, const __half* pkv, int P,
                            const __half* kvc, const int32_t* seq_start, __half* gkv, int gcap, int slot, __half* out,
                            int* err, cudaStream_t s);
// Token of step t for every row from the packed LM-head argmax (best[] is reset
// to 0), pad after an eos, and the fed-back position P + len + t.
void launch_decode_select(unsigned long long* best, int R, int t, int max_new, int eos, int pad, int V, int32_t* done,
                          int32_t* gen_tok, int32_t* gen_len, int32_t* next_tok, int32_t* pos,
                          const int32_t* seq_start, int P, int* err, cudaStream_t s);
void launch_patch_empty_rows(float* resid, const int32_t* last_idx, const float* prefix_last, int R, int d,
                             cudaStream_t s);
void launch_bias_f32(const uint16_t* b, int V, int Vpad, float* out, cudaStream_t s);
void launch_like_match(const int32_t* gen_tok, const int32_t* gen_len, int64_t S, int max_new, const int32_t* pattern,
                       int plen, int32_t* match, cudaStream_t s);
void launch_gather_rows_i32(const int32_t* src, int width, const int32_t* pos, int64_t n, int32_t* out,
                            cudaStream_t s);
// ---------------------------------------------------------------- pairs ---
// Device scratch of the Q4 self-join over S candidates (sizes in elements):
// keys, keys_tmp [S] u64; vals, vals_tmp, heads, counts [S] i32; head_excl,
// pair_off [S + 1] i64; group_start [S + 1] i64; hist [256 * tiles] i32,
// hist_off [256 * tiles + 1] i64 (tiles = ceil(S / 2048)); scan_tmp
// [2 * (ceil(max(S, 256 * tiles) / 2048) + 1)] i64.
struct SelfJoinScratch {
  uint64_t *keys, *keys_tmp;
  int32_t *vals, *vals_tmp, *heads, *counts, *hist;
  int64_t *head_excl, *pair_off, *group_start, *hist_off, *scan_tmp;
};
// Sort the candidates by key (stable), group them, and write pair_off: the
// exclusive scan, in candidate order, of each candidate's pair count (its
// group members after it); pair_off[S] is the number of pairs.
void launch_self_join_pairs_plan(const int64_t* key_col, const int32_t* ids, int64_t S, const SelfJoinScratch& w,
                                 cudaStream_t s);
// (pa[k], pb[k]) = the k-th pair (a < b, equal keys), ascending (a, b).
void launch_self_join_pairs_emit(const int32_t* ids, int64_t S, const SelfJoinScratch& w, int32_t* pa, int32_t* pb,
                                 cudaStream_t s);

// bits / per-block counts of the non-zero entries of an int32 flag array.
void launch_flag_mask(const int32_t* flags, int64_t n, uint32_t* bits, int32_t* block_counts, cudaStream_t s);

// Sets the thread-local message that aiq_last_error() returns.
void set_error_message(const char* msg);
// Records a failed launch; the next status check of the query reports it.
void set_launch_error(const char* what, cudaError_t e);
// Returns and clears the recorded launch failure (cudaSuccess if none).
cudaError_t take_launch_error(const char** what);

}  // namespace aiq
