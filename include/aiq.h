/* aiq.h - C-ABI of the unified AI-query library (libaiq.so), GB300 / sm_103a.
 *
 * One call runs a whole AI query on the GPU: relational predicate, stream
 * compaction of the surviving row ids, (optionally) a hash equi-join, packing
 * of every candidate row's tokens behind a shared prompt prefix, a decoder-only
 * transformer prefill over the packed variable-length batch, the label-logit
 * decision at each row's last position and the masked aggregate.  Only the
 * results cross PCIe (the paper's "H2D boundary consolidation", Section 3.3).
 *
 * Conventions for every entry point:
 *   - Returns an aiq_status; never aborts the process.  On failure
 *     aiq_last_error() describes the cause (thread-local string, valid until
 *     the next call on the same thread).
 *   - Calls are synchronous: results are on the host when the call returns.
 *   - Load calls COPY the caller's host buffers to the device; the caller keeps
 *     ownership of its buffers.  Tables, models and results belong to the
 *     library until their free call (or aiq_shutdown).
 *   - A context is bound to one device and is not thread-safe: serialise
 *     calls on one context.
 */
#ifndef AIQ_H
#define AIQ_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  AIQ_OK = 0,
  AIQ_ERR_INVALID_ARG = -1,  /* bad pointer, size, id, type or shape */
  AIQ_ERR_NOT_FOUND = -2,    /* unknown table / model / result handle */
  AIQ_ERR_OOM = -3,          /* device allocation failed or AIQ_DEVICE_BYTES_MAX exceeded */
  AIQ_ERR_CUDA = -4,         /* a CUDA runtime call failed */
  AIQ_ERR_CAPACITY = -5,     /* a fixed-capacity structure overflowed */
  AIQ_ERR_DEVICE_CHECK = -6, /* a kernel's own check failed (bounded wait expired, fp16 overflow) */
  AIQ_ERR_UNSUPPORTED = -7   /* valid input outside what this build implements */
} aiq_status;

typedef enum { AIQ_INT32 = 0, AIQ_INT64 = 1, AIQ_FLOAT32 = 2, AIQ_TOKENS = 3 } aiq_dtype;

/* One column of a table.  INT32 / INT64 / FLOAT32: `data` points to n_rows
 * values.  TOKENS (a tokenised text column, CSR): `data` points to int32 token
 * ids and `offsets` to n_rows + 1 non-decreasing int64 offsets into them, with
 * offsets[0] = 0.  Table 1 of the paper, FROM row: the table's arrays are
 * loaded into device memory once. */
typedef struct {
  const char* name;
  int32_t type; /* aiq_dtype */
  const void* data;
  const int64_t* offsets; /* TOKENS only */
} aiq_column;

/* Decoder shape.  Llama-style pre-norm blocks: RMSNorm, rotary embeddings
 * (half-split pairs), causal grouped-query attention, SwiGLU MLP, untied LM
 * head with a bias.  head_dim must be 32, 64 or 128; n_heads a multiple of
 * n_kv_heads; d_model, d_ffn multiples of 128. */
typedef struct {
  int32_t n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ffn, vocab;
  float rope_theta, rms_eps;
} aiq_model_config;

typedef enum { AIQ_LT = 0, AIQ_LE = 1, AIQ_GT = 2, AIQ_GE = 3, AIQ_EQ = 4, AIQ_NE = 5 } aiq_cmp;

/* One relational term `column op constant` (Table 1, WHERE row).  A query's
 * terms are conjoined.  INT32/INT64 columns compare with `ivalue`, FLOAT32
 * columns with `fvalue` (as float). */
typedef struct {
  int32_t column; /* index into the table's columns */
  int32_t op;     /* aiq_cmp */
  int64_t ivalue;
  double fvalue;
} aiq_pred;

typedef enum {
  AIQ_AGG_COUNT = 0,          /* COUNT(*) of rows decided "yes" (2 labels) */
  AIQ_AGG_ROW_IDS = 1,        /* ids of the "yes" rows, ascending, and their count */
  AIQ_AGG_GROUP_LABEL = 2,    /* GROUP BY predicted label COUNT(*), all labels */
  AIQ_AGG_GROUP_BUILD_KEY = 3, /* joins: GROUP BY build-side key COUNT(*) of "yes" rows */
  AIQ_AGG_SUM = 4              /* SUM(sum_column) over the "yes" rows, and their count (Fig. 2's
                                  masked reduction); integer columns sum exactly in int64 (wrapping
                                  on overflow), FLOAT32 columns in fp64 in a fixed order */
} aiq_agg;

enum {
  AIQ_FLAG_LOGITS = 1,          /* also return per-candidate label logits, ids and decisions */
  AIQ_FLAG_RELATIONAL_ONLY = 2  /* stop after the relational phase; return the candidates */
};

/* The AI part of a query (Fig. 2): each candidate row's prompt is
 * prefix ++ tokens(text_column); the label logits are read at its last
 * position.  With 2 labels the row is "yes" iff logit(label 0) > logit(label 1)
 * (strict); with more labels the prediction is the first index of the largest
 * logit. */
typedef struct {
  const aiq_pred* preds;
  int32_t n_preds;       /* 0..8 */
  int32_t text_column;   /* index of a TOKENS column */
  const int32_t* prefix; /* host, prefix_len token ids */
  int32_t prefix_len;
  const int32_t* label_ids; /* host, n_labels token ids (2..16) */
  int32_t n_labels;
  int32_t agg;   /* aiq_agg */
  int32_t flags; /* AIQ_FLAG_* */
  int32_t sum_column; /* AIQ_AGG_SUM: index of an INT32, INT64 or FLOAT32 column (else ignored) */
} aiq_select;

/* Result view.  Pointers are host memory owned by the result; valid until
 * aiq_result_free.  Absent outputs are NULL with a zero length. */
typedef struct {
  int64_t n_input_rows; /* rows scanned (probe side for joins) */
  int64_t n_candidates; /* rows that reached the language model */
  int64_t n_tokens;     /* prompt tokens of all candidates (prefix + row text each) */
  int64_t n_chunks;     /* token-budget chunks the prefill ran in */
  int64_t count;        /* number of "yes" rows (2 labels), else -1 */
  const int32_t* row_ids;
  int64_t n_row_ids;
  const int32_t* group_build_rows; /* GROUP_BUILD_KEY: ascending build row */
  const int64_t* group_keys;
  const int64_t* group_counts;
  int64_t n_groups;
  const int64_t* label_counts; /* [n_labels]: decisions per label */
  int32_t n_labels;
  /* AIQ_FLAG_LOGITS / AIQ_FLAG_RELATIONAL_ONLY */
  const int32_t* cand_row_ids;    /* [n_candidates] ascending (probe order for joins) */
  const int32_t* cand_build_rows; /* joins: matching build row per candidate */
  const float* label_logits;      /* [n_candidates, n_labels] */
  const int32_t* decisions;       /* [n_candidates] */
  /* device time of the phases (CUDA events on the library's stream) */
  float ms_relational, ms_prefill, ms_aggregate, ms_total;
  double prefill_flops; /* executed: 2*params per token + 4*Hq*hd*L per causal pair + head */
  int64_t n_launches;   /* CUDA kernels this query launched */
  int64_t n_prefill_tokens; /* tokens run through the decoder: the shared prefix once + every row's text */
  /* aiq_run_pair_select with AIQ_AGG_ROW_IDS: the B row of each yes pair (row_ids holds its A row) */
  const int32_t* row_ids_b;
  /* aiq_run_transform only (zero / NULL otherwise) */
  int32_t gen_max_new;        /* columns of gen_tokens: the generate spec's max_new_tokens */
  int64_t n_gen_rows;         /* rows of gen_tokens */
  const int32_t* gen_row_ids; /* [n_gen_rows] ascending table rows */
  const int32_t* gen_tokens;  /* [n_gen_rows, gen_max_new]: greedy tokens, the eos, then pad_id */
  const int32_t* gen_text_len; /* [n_gen_rows]: generated tokens before the eos (max_new without one) */
  float ms_decode;            /* device time of the decode steps (inside ms_prefill) */
  double decode_flops;        /* 2*params per decoded token + attention over cached keys + full LM head */
  int64_t n_decode_steps;     /* sum over prefill chunks of max_new_tokens */
  /* AIQ_AGG_SUM: the sum (sum_int for INT32 / INT64 columns, sum_float for FLOAT32); with
   * count == 0 it is 0 (SQL's NULL) */
  int64_t sum_int;
  double sum_float;
} aiq_result_view;

typedef struct aiq_ctx aiq_ctx;
typedef int64_t aiq_table;
typedef int64_t aiq_model;
typedef int64_t aiq_result_h;

/* Section 3 (opening): the whole AI query, relational operators and LLM
 * inference together, runs as one program on one accelerator.  A context is
 * that accelerator: CUDA device `device`, one stream on which every step of a
 * query is issued, and the device memory that holds the resident tables,
 * models and the query workspace.  Options come from the environment:
 * AIQ_DEVICE_BYTES_MAX caps the bytes the context may allocate (AIQ_ERR_OOM
 * beyond it).  *out is owned by the caller until aiq_shutdown.  Errors:
 * AIQ_ERR_INVALID_ARG (NULL out, no such device), AIQ_ERR_UNSUPPORTED (not an
 * sm_103 GPU), AIQ_ERR_CUDA (the device cannot be initialised). */
aiq_status aiq_init(int device, aiq_ctx** out);
/* Section 3 (opening): ends the context of aiq_init.  Frees every table,
 * model, result and buffer of the context; ctx is invalid afterwards.  NULL
 * is ignored. */
void aiq_shutdown(aiq_ctx* ctx);

/* Table 1, FROM row: copy n_cols columns of n_rows rows to the device.
 * n_rows must be < 2^31 (row ids are int32).  Token offsets are checked
 * (start at 0, non-decreasing, fewer than 2^31 tokens); token ids must be
 * non-negative here, and are checked against the model's vocabulary per query.
 * The copy has completed when the call returns: the caller may free or reuse
 * its buffers.  Errors: AIQ_ERR_INVALID_ARG (a check above, NULL data, an
 * unknown type), AIQ_ERR_UNSUPPORTED (2^31 tokens or more), AIQ_ERR_OOM,
 * AIQ_ERR_CUDA; on error nothing stays allocated. */
aiq_status aiq_load_table(aiq_ctx* ctx, const aiq_column* cols, int32_t n_cols, int64_t n_rows, aiq_table* out);
aiq_status aiq_free_table(aiq_ctx* ctx, aiq_table table);

/* Fig. 2: the semantic operator is a causal-LM forward pass whose weights
 * live on the accelerator beside the table; Section 3.2: the model is the AI
 * operator's template that the compiled program calls.  Copies a model's
 * weights (host bf16 bit patterns, uint16; the caller keeps its buffers) to
 * the device, where they stay resident until aiq_free_model.
 * Tensor order, linear weights in [out_features, in_features] layout:
 *   embed [V, d];
 *   per layer: attn_norm [d], wq [Hq*hd, d], wk [Hkv*hd, d], wv [Hkv*hd, d],
 *              wo [d, Hq*hd], mlp_norm [d], wg [f, d], wu [f, d], wd [d, f];
 *   final_norm [d], lm_head [V, d], lm_bias [V].
 * n_tensors = 1 + 9 * n_layers + 3.  Linear weights are held as fp16 tensor-core
 * operands (exact for every bf16 value of magnitude >= 2^-17; a weight above
 * the fp16 range gives AIQ_ERR_UNSUPPORTED). */
aiq_status aiq_load_model(aiq_ctx* ctx, const aiq_model_config* cfg, const void* const* bf16_tensors,
                          int32_t n_tensors, aiq_model* out);
aiq_status aiq_free_model(aiq_ctx* ctx, aiq_model model);

/* Table 2 Q1/Q2: SELECT <agg> FROM table WHERE <preds> AND AI(text) = yes.
 * Token ids of the prefix, labels and the candidate rows must be < vocab
 * (AIQ_ERR_INVALID_ARG otherwise).  model may be 0 with AIQ_FLAG_RELATIONAL_ONLY. */
aiq_status aiq_run_select(aiq_ctx* ctx, aiq_table table, aiq_model model, const aiq_select* q, aiq_result_h* out);

/* Section 4 datasets: probe JOIN build ON probe.key = build.key, with build
 * terms (e.g. movies.year >= 2010) and the probe-side select.  Build keys must
 * be unique INT64 values other than INT64_MIN (AIQ_ERR_INVALID_ARG otherwise);
 * probe keys may repeat or match nothing.  Candidates are the joined probe
 * rows in ascending probe order. */
aiq_status aiq_run_join_select(aiq_ctx* ctx, aiq_table build, int32_t build_key, const aiq_pred* build_preds,
                               int32_t n_build_preds, aiq_table probe, int32_t probe_key, aiq_model model,
                               const aiq_select* probe_side, aiq_result_h* out);

/* AI_TRANSFORM (Table 1: causal-LM forward with generative decoding, output
 * masked with a pad id; Table 2 Q3 and Q5).  Greedy decoding: every step
 * appends the first index of the largest full-vocabulary logit (final RMSNorm,
 * LM head, bias) at the row's last position.  After a row emits eos_id, its
 * remaining positions hold pad_id; eos_id < 0 disables the stop.
 * like_len > 0 adds Q5's filter: a row matches when the pattern occurs as a
 * contiguous run of its generated tokens before the eos (SQL LIKE '%...%' on
 * token ids); like_len == 0 with a non-NULL like_tokens matches every row. */
typedef struct {
  int32_t max_new_tokens;     /* 1..4096 */
  int32_t eos_id;             /* -1: none */
  int32_t pad_id;
  const int32_t* like_tokens; /* host; NULL: no LIKE filter (Q3 form) */
  int32_t like_len;           /* 0..256 */
  int32_t flags;              /* AIQ_GEN_* */
} aiq_generate;

enum {
  AIQ_GEN_MATCH_TOKENS = 1 /* with LIKE: also return the matching rows' tokens (the "debug outputs") */
};

/* Table 2 Q3: SELECT AI_TRANSFORM(text, prefix) FROM table WHERE <preds>:
 *   gen_row_ids = the candidate rows, gen_tokens / gen_text_len per row, count = -1.
 * Table 2 Q5: SELECT COUNT(*) ... WHERE <preds> AND AI_TRANSFORM(...) LIKE '%p%':
 *   count = matching rows, row_ids = their ids; with AIQ_GEN_MATCH_TOKENS the
 *   gen_* arrays hold the matching rows only.
 * Uses q's preds, text_column and prefix; its labels, agg and flags are ignored.
 * Token ids of the prefix and the rows must be < vocab; pad_id and eos_id too
 * (when set).  The whole generation runs on the device: only the results
 * cross PCIe. */
aiq_status aiq_run_transform(aiq_ctx* ctx, aiq_table table, aiq_model model, const aiq_select* q,
                             const aiq_generate* gen, aiq_result_h* out);

/* Table 2 Q4: SELECT A.text, B.text, AI_IF([A.text, B.text]) FROM table A
 * CROSS JOIN table B WHERE <preds> AND A.key = B.key AND A.row < B.row.
 * The terms filter the table before it is joined with itself (both sides);
 * key_column is an INT64 column; each pair (a, b) of selected rows with equal
 * keys and a < b (the row index is the review id) is one candidate, in
 * ascending (a, b) order, and its prompt is prefix ++ text(a) ++ text(b).
 * The pairs are formed on the device: only the table crosses PCIe (§4.3).
 * Candidates are pairs: n_candidates = number of pairs; with AIQ_FLAG_LOGITS
 * cand_row_ids / cand_build_rows hold every pair's A / B row with its logits
 * and decision; AIQ_AGG_COUNT gives the yes pairs' count, AIQ_AGG_ROW_IDS also
 * their A rows (row_ids) and B rows (row_ids_b).  2 labels.  More than
 * 2^31 - 1 pairs gives AIQ_ERR_CAPACITY. */
aiq_status aiq_run_pair_select(aiq_ctx* ctx, aiq_table table, int32_t key_column, aiq_model model,
                               const aiq_select* q, aiq_result_h* out);

/* Section 3.3 (H2D boundary consolidation): only a query's final results
 * cross back to the host, never its masks, activations or logits (the
 * per-candidate logits only on request, the paper's debug outputs of Table 2
 * Q5).  Fills *out with host pointers to those results; they stay valid until
 * aiq_result_free of the same handle.  Errors: AIQ_ERR_NOT_FOUND (unknown
 * handle), AIQ_ERR_INVALID_ARG (NULL out). */
aiq_status aiq_result(aiq_ctx* ctx, aiq_result_h result, aiq_result_view* out);
/* Section 3.3: releases the host copy of a query's results; the view's
 * pointers are invalid afterwards.  AIQ_ERR_NOT_FOUND for an unknown handle. */
aiq_status aiq_result_free(aiq_ctx* ctx, aiq_result_h result);

/* Thread-local description of the last failure on this thread ("" if none). */
const char* aiq_last_error(void);

/* Options: "token_budget" (max packed tokens per prefill chunk, default
 * 131072), "profile" (0/1: time every GEMM launch with CUDA events),
 * "gemm_pair" (0/1, default 1: 256 x 256 GEMM tiles on CTA pairs where
 * N % 256 == 0 and M >= 512; also selects them for aiq_op_gemm with bn = 256),
 * "attention_tc" (0/1, default 1: tcgen05 attention where the head shape
 * allows), "mlp_split" (read by aiq_load_model; 1: the model's MLP GEMMs
 * take their activations as two fp16 terms, fp16(v) and fp16(v - fp16(v)),
 * against weights stored twice along K, about twice the MLP's tensor work and
 * weight memory for a smaller error; 0: one fp16 term; default -1: on for
 * models of at least 32 layers and d_model 4096, whose label logits otherwise
 * drift past the 2e-2 margin tolerance on a few rows),
 * "decode_rows" (aiq_run_transform: rows per prefill chunk, which
 * decode together, default 4096; the chunk's token budget grows to fit them,
 * up to 2^20 tokens and 32 GB of cached prompt keys/values), "device_bytes_max"
 * (the context's device byte cap, as AIQ_DEVICE_BYTES_MAX at aiq_init; <= 0
 * lifts it; memory already held stays, only further growth is refused with
 * AIQ_ERR_OOM). */
aiq_status aiq_set_option(aiq_ctx* ctx, const char* name, int64_t value);

/* The context's CUDA stream (a cudaStream_t), for callers that time the
 * library's work with their own events. */
void* aiq_stream(aiq_ctx* ctx);

/* Per-kernel-class device time accumulated while "profile" is on. */
typedef struct {
  const char* name;
  int64_t launches;
  double total_ms;
  double flops; /* algorithmic FLOPs of those launches */
  double bytes; /* algorithmic bytes of those launches */
} aiq_kernel_stat;
/* Writes up to `max` entries; *n_out receives the number written. */
aiq_status aiq_kernel_stats(aiq_ctx* ctx, aiq_kernel_stat* out, int32_t max, int32_t* n_out);
aiq_status aiq_reset_kernel_stats(aiq_ctx* ctx);

#ifdef __cplusplus
}
#endif
#endif /* AIQ_H */
