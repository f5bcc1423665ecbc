/* aiq_ops.h - step-level C-ABI of libaiq.so: the prefill kernels one at a time.
 *
 * These entry points run one step of the query's prefill on caller-owned
 * DEVICE buffers (plain device pointers, element counts), on the context's
 * stream, and synchronise before returning.  They exist so that each kernel
 * can be checked on its own; the whole query uses the same kernels through
 * aiq_run_select / aiq_run_join_select.  All return aiq_status; a kernel's
 * own check (fp16 overflow, an expired bounded wait) gives
 * AIQ_ERR_DEVICE_CHECK.  The caller keeps ownership of every buffer.
 */
#ifndef AIQ_OPS_H
#define AIQ_OPS_H

#include <stdint.h>

#include "aiq.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  AIQ_EPI_F16 = 0,       /* out fp16 [M, N] = A B^T */
  AIQ_EPI_ROPE_F16 = 1,  /* as F16, then rotary embedding on columns < rope_cols */
  AIQ_EPI_RESID_F32 = 2, /* out fp32 [M, N] += A B^T (residual stream update) */
  AIQ_EPI_SWIGLU_F16 = 3, /* B rows interleave gate/up blocks of bn/2: out fp16 [M, N/2] = silu(g) * u */
  AIQ_EPI_RESID_ADD_F32 = 5 /* as RESID_F32, the add done by TMA reduce-add tiles (out 16-byte aligned,
                               ldo a multiple of 4) */
} aiq_epilogue;

/* A decoder linear layer on the tensor cores: A fp16 [M, K] (row pitch lda
 * elements) times B fp16 [N, K] (row pitch ldb; nn.Linear [out, in] layout),
 * fp32 accumulation, then the epilogue.  bn = 128 or 256 is the output tile
 * width: N % bn == 0, K % 64 == 0, rows 16-byte aligned.
 * ROPE: `positions` int32 [M] (device), `rope_cos`/`rope_sin` fp32
 * [max_pos, head_dim/2] (see aiq_op_rope_table); pairs (i, i + head_dim/2) of
 * each head starting below rope_cols are rotated (the q and k heads of a
 * fused QKV output).  SwiGLU MLP and rotary embeddings follow the decoder
 * reading stated in aiq_model_config. */
aiq_status aiq_op_gemm(aiq_ctx* ctx, const void* A, int64_t lda, const void* B, int64_t ldb, int32_t M, int32_t N,
                       int32_t K, int32_t bn, int32_t epilogue, void* out, int64_t ldo, const int32_t* positions,
                       const float* rope_cos, const float* rope_sin, int32_t rope_cols, int32_t head_dim);

/* cos/sin of pos * theta^(-2i/head_dim), i < head_dim/2, pos < max_pos, computed
 * in fp64 and stored fp32 [max_pos, head_dim/2] (device). */
aiq_status aiq_op_rope_table(aiq_ctx* ctx, float* rope_cos, float* rope_sin, int32_t max_pos, int32_t head_dim,
                             float theta);

/* out fp16 [T, d] = x / sqrt(mean(x^2) + eps) * g, x fp32 [T, d], g bf16 [d]. */
aiq_status aiq_op_rmsnorm(aiq_ctx* ctx, const float* x, int64_t T, int32_t d, const uint16_t* g, float eps,
                          void* out);

/* Causal grouped-query attention over a packed variable-length batch.
 * qkv fp16 [T, (Hq + 2 Hkv) * hd]: q heads, then k heads, then v heads, with
 * rotary embeddings already applied.  seq_start int32 [n_seqs + 1] (device):
 * sequence i occupies rows [seq_start[i], seq_start[i+1]); seq_start[n_seqs]
 * = T.  Query head h reads key/value head h / (Hq / Hkv).  prefix_kv
 * (optional, P > 0): fp16 [P, 2 Hkv hd] keys then values of a shared prompt
 * prefix at positions before every sequence, which every query also attends
 * (the prefix's K/V are computed once per query and reused by every row).
 * out fp16 [T, Hq * hd].  hd in {32, 64, 128}. */
aiq_status aiq_op_attention(aiq_ctx* ctx, const void* qkv, int64_t T, const int32_t* seq_start, int32_t n_seqs,
                            int32_t Hq, int32_t Hkv, int32_t hd, const void* prefix_kv, int32_t P, void* out);

/* One decode step of causal grouped-query attention (AI_TRANSFORM, Table 1:
 * generative decoding; each row attends every earlier token of its own
 * sequence).  R rows, one new token each: qkv fp16 [R, (Hq + 2 Hkv) * hd]
 * (rotary embeddings applied).  Row r's keys/values, every cache fp16 with
 * rows of [2 Hkv hd] (keys, then values):
 *   prefix_kv [P] shared by every row (may be NULL when P == 0);
 *   own_kv rows [seq_start[r], seq_start[r+1]) (seq_start int32 [R + 1], device);
 *   gen_kv [R, gen_cap] slots 0 .. slot of row r, where slot `slot` first
 *   receives this step's key and value (written by the call).
 * out fp16 [R, Hq * hd].  hd in {32, 64, 128}, Hq / Hkv <= 8.  All pointers are
 * device memory owned by the caller; the call synchronises its stream. */
aiq_status aiq_op_decode_attention(aiq_ctx* ctx, const void* qkv, int32_t R, int32_t Hq, int32_t Hkv, int32_t hd,
                                   const void* prefix_kv, int32_t P, const void* own_kv, const int32_t* seq_start,
                                   void* gen_kv, int32_t gen_cap, int32_t slot, void* out);

/* One relational term for aiq_filter_compact_static: `column op constant` on a
 * caller-owned device column of n_rows values (16-byte aligned).  INT32 and
 * INT64 columns compare with `ivalue`, FLOAT32 columns with `fvalue`. */
typedef struct {
  const void* column; /* device pointer */
  int32_t type;       /* AIQ_INT32, AIQ_INT64 or AIQ_FLOAT32 */
  int32_t op;         /* aiq_cmp */
  int64_t ivalue;
  double fvalue;
} aiq_term;

/* Filter and compact without allocating: the ids (ascending, int32) of the rows
 * of caller-owned device columns that satisfy every term, written to ids_out
 * (device, room for n_rows ids), and their number to *count_out (device int64).
 * The paper has no counterpart: this is for callers that must not allocate
 * device memory while they run (a worker confined to a fixed device arena, an
 * operator inside another engine's allocation-free loop, a latency-bound path
 * that cannot take cudaMalloc's implicit synchronisation or its failure under
 * memory pressure).  It runs the same kernels as aiq_run_select's
 * relational phase, asynchronously on `stream` (a cudaStream_t; NULL = the
 * legacy default stream), with their scratch in one static device array of
 * about 2.1 MB that every GPU loading the library keeps until the process exits.
 *   - At most 16,777,216 rows per call (AIQ_ERR_CAPACITY beyond), 0..8 terms.
 *   - No cudaMalloc, cudaFree or allocating library call is made.  The first
 *     call on a device looks up the array's device address once
 *     (cudaGetSymbolAddress) with that device current; make that first call
 *     before any stream capture.  The address is cached for the life of the
 *     process: after a cudaDeviceReset of a device, do not call this entry
 *     point on that device again.
 *   - All calls share the one array: two calls whose work overlaps on the GPU
 *     (different streams, or different host threads on one device) race and
 *     both results are undefined.  Calls ordered on one stream are safe; each
 *     call rewrites every scratch word it reads.
 *   - n_rows == 0 writes 0 to *count_out and nothing to ids_out.
 *   - Errors are returned as aiq_status, described by aiq_last_error(); a
 *     failed kernel launch gives AIQ_ERR_CUDA and leaves ids_out and
 *     *count_out undefined. */
aiq_status aiq_filter_compact_static(const aiq_term* terms, int32_t n_terms, int64_t n_rows, int32_t* ids_out,
                                     int64_t* count_out, void* stream);

/* Self-test of the device-side failure detection that every pipelined kernel
 * of the library uses.  One CTA of two warps waits on an mbarrier phase that
 * nothing completes: warp 0 with a limit of limit_ns, warp 1 with four times
 * that, both through the same bounded wait as the kernels.  Warp 0's wait runs
 * out, records the timeout and raises the CTA's abort flag, on which warp 1
 * returns without waiting out its own limit.  The call then returns
 * AIQ_ERR_DEVICE_CHECK ("a kernel's bounded wait expired"), and the context
 * stays usable: the device error word is cleared and no CUDA error is left.
 * limit_ns in [1000, 1000000000]; anything else gives AIQ_ERR_INVALID_ARG. */
aiq_status aiq_op_wait_expiry_selftest(aiq_ctx* ctx, uint64_t limit_ns);

#ifdef __cplusplus
}
#endif
#endif /* AIQ_OPS_H */
