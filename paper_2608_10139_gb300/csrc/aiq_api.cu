// C-ABI of the unified AI-query library: contexts, device-resident tables and
// models, the query planner and the step-level ops.
//
// A query is one pipeline on one CUDA stream (the paper's single compiled
// program, Section 3): predicate + compaction (+ hash join), token packing,
// chunked decoder prefill, label-logit decision, masked aggregate.  The host
// reads back only control scalars between phases (survivor count, token
// count, the chunk table) and the final results; no intermediate array
// crosses PCIe (Section 3.3, H2D boundary consolidation).
#include <algorithm>
#include <cstdlib>
#include <cstring>
#include <map>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "aiq.h"
#include "aiq_ops.h"
#include "common.cuh"
#include "kernels.h"

using namespace aiq;

namespace {

thread_local std::string g_err;

aiq_status fail(aiq_status st, const std::string& msg) {
  g_err = msg;
  return st;
}

#define CUDA_TRY(x)                                                                         \
  do {                                                                                      \
    cudaError_t e_ = (x);                                                                   \
    if (e_ != cudaSuccess) {                                                                \
      cudaGetLastError();                                                                   \
      return fail(AIQ_ERR_CUDA, std::string(#x) + ": " + cudaGetErrorString(e_));          \
    }                                                                                       \
  } while (0)

#define AIQ_TRY(x)                 \
  do {                             \
    aiq_status s_ = (x);           \
    if (s_ != AIQ_OK) return s_;   \
  } while (0)

struct DevBuf {
  void* p = nullptr;
  size_t bytes = 0;
};

struct ColD {
  std::string name;
  int32_t type = 0;
  void* data = nullptr;
  int64_t* offsets = nullptr;
  size_t bytes = 0;
  int64_t max_len = 0;   // TOKENS: longest row
  int64_t min_len = 0;   // TOKENS: shortest row
  int64_t max_id = -1;   // TOKENS: largest token id
};

struct TableD {
  int64_t n_rows = 0;
  std::vector<ColD> cols;
};

struct LayerD {
  uint16_t* attn_norm = nullptr;
  uint16_t* mlp_norm = nullptr;
  __half* wqkv = nullptr;  // [(Hq + 2 Hkv) hd, d]
  __half* wo = nullptr;    // [d, Hq hd]
  __half* wgu = nullptr;   // [2 f, d] ([2 f, 2 d] with mlp_split), gate/up interleaved in blocks of bn_gu / 2 rows
  __half* wd = nullptr;    // [d, f] ([d, 2 f] with mlp_split)
};

struct ModelD {
  aiq_model_config cfg{};
  uint16_t* embed = nullptr;
  uint16_t* final_norm = nullptr;
  uint16_t* lm_head = nullptr;
  uint16_t* lm_bias = nullptr;
  std::vector<LayerD> layers;
  std::vector<DevBuf> allocs;
  int bn_qkv = 128, bn_o = 128, bn_gu = 128, bn_d = 128;
  // two-term MLP activations: the gate/up and down GEMMs run over K = 2d and
  // 2f against their weights stored twice along K, with the activation as
  // fp16(v) followed by fp16(v - fp16(v))
  bool mlp_split = false;
  DevBuf rope_cos, rope_sin;
  int rope_max_pos = 0;
  double linear_flops_per_token = 0;
  // full-vocabulary LM head for generation, made on first use: fp16 [vpad, d]
  // (zero rows past the vocabulary) and an fp32 bias with -inf past it
  __half* lm_f16 = nullptr;
  float* lm_bias_f32 = nullptr;
  int vpad = 0;
};

struct ResultH {
  aiq_result_view v{};
  std::vector<int32_t> row_ids, group_rows, cand_ids, cand_build, decisions;
  std::vector<int64_t> group_keys, group_counts, label_counts;
  std::vector<float> logits;
  std::vector<int32_t> gen_ids, gen_tok, gen_len, row_ids_b;
  uint64_t sum_bits = 0;  // AIQ_AGG_SUM: int64 or double bits
  bool sum_is_float = false;
  int32_t gen_max_new = 0;
};

struct ProfRec {
  const char* name;
  cudaEvent_t a, b;
  double flops, bytes;
};

struct StatAcc {
  int64_t launches = 0;
  double ms = 0, flops = 0, bytes = 0;
};

}  // namespace

void aiq::set_error_message(const char* msg) { g_err = msg ? msg : ""; }

namespace {
thread_local cudaError_t g_launch_err = cudaSuccess;
thread_local std::string g_launch_what;
}  // namespace

void aiq::set_launch_error(const char* what, cudaError_t e) {
  if (g_launch_err == cudaSuccess) {
    g_launch_err = e;
    g_launch_what = what ? what : "";
  }
}

cudaError_t aiq::take_launch_error(const char** what) {
  const cudaError_t e = g_launch_err;
  g_launch_err = cudaSuccess;
  if (what) *what = g_launch_what.c_str();
  return e;
}

namespace {
// NVTX ranges (host issue time) that name a query's phases for profilers:
// "relational", "prefill" (with one "prefix" and one "chunk" range per token
// chunk inside it) and "aggregate".  begin() closes the previous phase.
class NvtxPhase {
 public:
  NvtxPhase() = default;
  explicit NvtxPhase(const char* name) { begin(name); }
  ~NvtxPhase() { end(); }
  void begin(const char* name) {
    end();
    nvtxRangePushA(name);
    open_ = true;
  }
  void end() {
    if (open_) nvtxRangePop();
    open_ = false;
  }

 private:
  bool open_ = false;
};
}  // namespace

struct aiq_ctx {
  int device = 0;
  int num_sms = 0;
  cudaStream_t stream = nullptr;
  int* d_err = nullptr;
  int64_t* h_pin = nullptr;  // pinned staging for control scalars
  size_t bytes_max = SIZE_MAX;
  size_t bytes_used = 0;
  int64_t next_handle = 1;
  std::map<int64_t, TableD> tables;
  std::map<int64_t, ModelD> models;
  std::map<int64_t, ResultH> results;
  std::map<std::string, DevBuf> ws;
  int64_t token_budget = 131072;
  bool profile = false;
  bool gemm_pair = true;  // CTA-pair (cta_group::2) GEMM tiles where the shape allows
  bool attention_tc = true;  // tcgen05 attention where the head shape allows
  // models loaded from now on: two-term MLP activations (K-doubled MLP GEMMs);
  // -1: for models of at least 32 layers and d_model 4096, where the one-term
  // fp16 path's label-logit error reaches the 2e-2 parity tolerance
  int mlp_split = -1;
  int64_t decode_rows = 4096;  // generation: target rows per prefill chunk (= decode batch)
  std::vector<ProfRec> prof;
  std::vector<cudaEvent_t> ev_pool;
  std::map<std::string, StatAcc> stats;
  std::vector<std::string> stat_names;
  int64_t launches = 0;  // kernels launched by the current query
};

namespace {

// ------------------------------------------------------------ allocation ---

aiq_status dalloc(aiq_ctx* c, void** p, size_t bytes) {
  bytes = std::max<size_t>(bytes, 256);
  if (c->bytes_used + bytes > c->bytes_max)
    return fail(AIQ_ERR_OOM, "device byte cap AIQ_DEVICE_BYTES_MAX exceeded (" + std::to_string(c->bytes_used + bytes) +
                                 " > " + std::to_string(c->bytes_max) + ")");
  cudaError_t e = cudaMalloc(p, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    *p = nullptr;
    return fail(AIQ_ERR_OOM, std::string("cudaMalloc(") + std::to_string(bytes) + "): " + cudaGetErrorString(e));
  }
  c->bytes_used += bytes;
  return AIQ_OK;
}

void dfree(aiq_ctx* c, void* p, size_t bytes) {
  if (!p) return;
  cudaFree(p);
  c->bytes_used -= std::max<size_t>(bytes, 256);
}

// Grow-only named workspace buffer.
template <typename T>
aiq_status ws(aiq_ctx* c, const char* name, size_t count, T** out) {
  size_t bytes = std::max<size_t>(count * sizeof(T), 256);
  DevBuf& b = c->ws[name];
  if (b.bytes < bytes) {
    if (b.p) {
      cudaStreamSynchronize(c->stream);
      dfree(c, b.p, b.bytes);
      b.p = nullptr;
      b.bytes = 0;
    }
    size_t want = bytes + bytes / 4;
    void* p = nullptr;
    if (dalloc(c, &p, want) != AIQ_OK) AIQ_TRY(dalloc(c, &p, want = bytes));
    b.p = p;
    b.bytes = want;
  }
  *out = static_cast<T*>(b.p);
  return AIQ_OK;
}

aiq_status sync_and_check(aiq_ctx* c) {
  const char* what = nullptr;
  const cudaError_t le = take_launch_error(&what);
  if (le != cudaSuccess) {
    cudaGetLastError();
    return fail(AIQ_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(le));
  }
  CUDA_TRY(cudaGetLastError());
  CUDA_TRY(cudaStreamSynchronize(c->stream));
  int err = 0;
  CUDA_TRY(cudaMemcpy(&err, c->d_err, sizeof(int), cudaMemcpyDeviceToHost));
  if (err) {
    // cleared on the context's stream, ordered before the next call's kernels
    CUDA_TRY(cudaMemsetAsync(c->d_err, 0, sizeof(int), c->stream));
    if (err & (DEVERR_DUP_BUILD_KEY | DEVERR_SENTINEL_KEY))
      return fail(AIQ_ERR_INVALID_ARG, "join build keys must be unique and differ from INT64_MIN");
    if (err & DEVERR_HASH_FULL) return fail(AIQ_ERR_CAPACITY, "hash table probe sequence exhausted");
    if (err & DEVERR_TIMEOUT) return fail(AIQ_ERR_DEVICE_CHECK, "a kernel's bounded wait expired");
    if (err & DEVERR_FP16_RANGE) return fail(AIQ_ERR_DEVICE_CHECK, "an activation left the fp16 range (or was NaN)");
    if (err & DEVERR_BOUNDS)
      return fail(AIQ_ERR_DEVICE_CHECK, "an index failed its bounds check (e.g. no finite logit for a greedy step)");
    return fail(AIQ_ERR_DEVICE_CHECK, "device check failed (code " + std::to_string(err) + ")");
  }
  return AIQ_OK;
}

// Reads `n` int64 values from the device after synchronising the stream.
aiq_status read_i64(aiq_ctx* c, const int64_t* dev, int64_t n, int64_t* host) {
  CUDA_TRY(cudaMemcpyAsync(host, dev, n * sizeof(int64_t), cudaMemcpyDeviceToHost, c->stream));
  return sync_and_check(c);
}

// ------------------------------------------------------------- profiling ---

cudaEvent_t take_event(aiq_ctx* c) {
  if (!c->ev_pool.empty()) {
    cudaEvent_t e = c->ev_pool.back();
    c->ev_pool.pop_back();
    return e;
  }
  cudaEvent_t e;
  cudaEventCreate(&e);
  return e;
}

struct ProfScope {
  aiq_ctx* c;
  const char* name;
  double flops, bytes;
  cudaEvent_t a = nullptr;
  ProfScope(aiq_ctx* c_, const char* n, double f, double b) : c(c_), name(n), flops(f), bytes(b) {
    if (c->profile) {
      a = take_event(c);
      cudaEventRecord(a, c->stream);
    }
  }
  ~ProfScope() {
    if (c->profile) {
      cudaEvent_t b2 = take_event(c);
      cudaEventRecord(b2, c->stream);
      c->prof.push_back({name, a, b2, flops, bytes});
    }
  }
};

void collect_profile(aiq_ctx* c) {
  if (c->prof.empty()) return;
  cudaStreamSynchronize(c->stream);
  for (auto& r : c->prof) {
    float ms = 0;
    cudaEventElapsedTime(&ms, r.a, r.b);
    StatAcc& s = c->stats[r.name];
    s.launches += 1;
    s.ms += ms;
    s.flops += r.flops;
    s.bytes += r.bytes;
    c->ev_pool.push_back(r.a);
    c->ev_pool.push_back(r.b);
  }
  c->prof.clear();
}

inline void counted(aiq_ctx* c, int n) { c->launches += n; }

// k_algo: the product's own depth when the GEMM runs over a two-term operand
// (K = 2 k_algo); the statistics count the algorithmic FLOPs and bytes.
aiq_status gemm(aiq_ctx* c, const char* name, const __half* A, int64_t lda, const __half* B, int64_t ldb, int M, int N,
                int K, int bn, const GemmEpilogue& ep, int k_algo = 0) {
  const double out_bytes =
      (ep.kind == EPI_RESID_F32 || ep.kind == EPI_RESID_ADD ? 8.0 : (ep.kind == EPI_SWIGLU_F16 ? 1.0 : 2.0)) * M * N;
  const double Ka = k_algo > 0 ? k_algo : K;
  ProfScope ps(c, name, 2.0 * M * N * Ka, 2.0 * (double(M) * Ka + double(N) * Ka) + out_bytes);
  const bool pair = c->gemm_pair && bn == 256 && M >= 512;
  int e = gemm_f16_tcgen05(A, lda, B, ldb, M, N, K, bn, pair, ep, c->num_sms, c->stream);
  if (M > 0) counted(c, 1);
  if (e != 0)
    return fail(AIQ_ERR_CUDA, std::string("tcgen05 GEMM launch: ") + cudaGetErrorString(static_cast<cudaError_t>(e)));
  return AIQ_OK;
}

// Causal GQA attention over a packed chunk: the work list, then the tcgen05
// kernel (head_dim 64/128) or the mma.sync kernel.
aiq_status attention(aiq_ctx* c, const __half* qkv, int64_t T, int64_t n_seqs, const int32_t* seq_start,
                     int32_t* tile_seq, int32_t* tile_q0, int32_t* n_tiles, int Hq, int Hkv, int hd,
                     const __half* pkv, int P, __half* out) {
  const bool tc = c->attention_tc && attention_tc_supported(hd, Hq, Hkv);
  const int tq = tc ? attention_tc_tile_tokens(Hq, Hkv) : 64;
  const int n_tiles_max = static_cast<int>((T + tq - 1) / tq + n_seqs);
  launch_attn_tiles(seq_start, static_cast<int32_t>(n_seqs), tq, tile_seq, tile_q0, n_tiles, c->stream);
  counted(c, 1);
  ProfScope p(c, "attention", 0, 0);
  if (tc) {
    const int e = launch_attention_tc(qkv, T, seq_start, tile_seq, tile_q0, n_tiles_max, n_tiles, Hq, Hkv, hd, pkv, P,
                                      out, c->d_err, c->num_sms, c->stream);
    if (e != 0)
      return fail(AIQ_ERR_CUDA, std::string("tcgen05 attention launch: ") +
                                    cudaGetErrorString(static_cast<cudaError_t>(e)));
  } else {
    launch_attention(qkv, T, seq_start, tile_seq, tile_q0, n_tiles_max, n_tiles, Hq, Hkv, hd, pkv, P, out, c->d_err,
                     c->stream);
  }
  counted(c, T > 0 && n_seqs > 0);
  return AIQ_OK;
}

// ------------------------------------------------------------ validation ---

aiq_status make_pred_set(const TableD& t, const aiq_pred* preds, int32_t n, PredSet* ps) {
  if (n < 0 || n > kMaxPreds) return fail(AIQ_ERR_INVALID_ARG, "n_preds must be 0..8");
  if (n > 0 && !preds) return fail(AIQ_ERR_INVALID_ARG, "preds is NULL");
  ps->n = n;
  for (int i = 0; i < n; ++i) {
    const aiq_pred& p = preds[i];
    if (p.column < 0 || p.column >= static_cast<int32_t>(t.cols.size()))
      return fail(AIQ_ERR_INVALID_ARG, "predicate column index out of range");
    const ColD& col = t.cols[p.column];
    if (col.type == AIQ_TOKENS) return fail(AIQ_ERR_INVALID_ARG, "predicate on a TOKENS column");
    if (p.op < AIQ_LT || p.op > AIQ_NE) return fail(AIQ_ERR_INVALID_ARG, "unknown comparison operator");
    ps->p[i] = PredDev{col.data, col.type, p.op, p.ivalue, p.fvalue};
  }
  return AIQ_OK;
}

ResultH& new_result(aiq_ctx* c, aiq_result_h* out) {
  const int64_t h = c->next_handle++;
  *out = h;
  return c->results[h];
}

// ----------------------------------------------------- relational phase ---

// Predicate (+ probe) over `t`, compaction into ids (and payload).  Returns S.
aiq_status filter_compact(aiq_ctx* c, const TableD& t, const PredSet& ps, const ProbeSpec& probe, const char* tag,
                          int64_t* S_out, int32_t** ids_out, int32_t** payload_out) {
  const int64_t n = t.n_rows;
  const int64_t nb = (n + kRowsPerBlock - 1) / kRowsPerBlock;
  std::string b = tag;
  uint32_t* bits;
  int32_t* bcnt;
  int64_t* boff;
  AIQ_TRY(ws(c, (b + ".bits").c_str(), std::max<int64_t>(nb, 1) * (kRowsPerBlock / 32), &bits));
  AIQ_TRY(ws(c, (b + ".bcnt").c_str(), std::max<int64_t>(nb, 1), &bcnt));
  AIQ_TRY(ws(c, (b + ".boff").c_str(), nb + 1, &boff));
  int64_t* scan_tmp;
  AIQ_TRY(ws(c, (b + ".scan").c_str(), 2 * (nb / kRowsPerBlock + 2), &scan_tmp));
  ProbeSpec pr = probe;
  if (pr.keys) {
    AIQ_TRY(ws(c, (b + ".match").c_str(), std::max<int64_t>(n, 1), &pr.match_out));
  }
  {
    ProfScope p(c, "predicate_mask", 0, 0);
    launch_predicate_mask(ps, pr, n, bits, bcnt, c->d_err, c->stream);
    counted(c, n > 0);
  }
  {
    ProfScope p(c, "scan_tiles", 0, 0);
    launch_scan_lengths(bcnt, nb, boff, scan_tmp, c->stream);
    counted(c, nb > 0 ? 3 : 0);
  }
  AIQ_TRY(read_i64(c, boff + nb, 1, c->h_pin));
  const int64_t S = c->h_pin[0];
  int32_t* ids;
  AIQ_TRY(ws(c, (b + ".ids").c_str(), std::max<int64_t>(S, 1), &ids));
  int32_t* pay = nullptr;
  if (pr.keys) AIQ_TRY(ws(c, (b + ".payload").c_str(), std::max<int64_t>(S, 1), &pay));
  {
    ProfScope p(c, "compact", 0, 0);
    launch_compact(bits, boff, n, ids, pr.match_out, pay, c->stream);
    counted(c, n > 0);
  }
  *S_out = S;
  *ids_out = ids;
  if (payload_out) *payload_out = pay;
  return AIQ_OK;
}

// --------------------------------------------------------- prefill phase ---

aiq_status ensure_rope(aiq_ctx* c, ModelD& m, int max_pos) {
  if (m.rope_max_pos >= max_pos) return AIQ_OK;
  const int want = std::max(max_pos, 2048);
  const size_t bytes = static_cast<size_t>(want) * (m.cfg.head_dim / 2) * sizeof(float);
  if (m.rope_cos.p) {
    CUDA_TRY(cudaStreamSynchronize(c->stream));
    dfree(c, m.rope_cos.p, m.rope_cos.bytes);
    dfree(c, m.rope_sin.p, m.rope_sin.bytes);
    m.rope_cos = m.rope_sin = DevBuf{};
    m.rope_max_pos = 0;
  }
  AIQ_TRY(dalloc(c, &m.rope_cos.p, bytes));
  m.rope_cos.bytes = bytes;
  AIQ_TRY(dalloc(c, &m.rope_sin.p, bytes));
  m.rope_sin.bytes = bytes;
  launch_rope_table(static_cast<float*>(m.rope_cos.p), static_cast<float*>(m.rope_sin.p), want, m.cfg.head_dim,
                    m.cfg.rope_theta, c->stream);
  counted(c, 1);
  m.rope_max_pos = want;
  return AIQ_OK;
}

struct PrefillBufs {
  int32_t *tok, *pos, *seq_start, *last_idx, *tile_seq, *tile_q0, *n_tiles, *last_compact;
  float *resid, *resid_last;
  float* ss_attn;  // per-128-column sums of squares of the residual, [T][d / 128]
  __half *xn, *qkv, *att, *act;
};

aiq_status prefill_bufs(aiq_ctx* c, const ModelD& m, int64_t B, int64_t max_rows, PrefillBufs* pb) {
  const aiq_model_config& g = m.cfg;
  const int64_t nqkv = static_cast<int64_t>(g.n_heads + 2 * g.n_kv_heads) * g.head_dim;
  AIQ_TRY(ws(c, "pf.tok", B, &pb->tok));
  AIQ_TRY(ws(c, "pf.pos", B, &pb->pos));
  AIQ_TRY(ws(c, "pf.seq_start", B + 1, &pb->seq_start));
  AIQ_TRY(ws(c, "pf.last", B, &pb->last_idx));
  AIQ_TRY(ws(c, "pf.tile_seq", B / 8 + B + 1, &pb->tile_seq));
  AIQ_TRY(ws(c, "pf.tile_q0", B / 8 + B + 1, &pb->tile_q0));
  AIQ_TRY(ws(c, "pf.n_tiles", 1, &pb->n_tiles));
  AIQ_TRY(ws(c, "pf.resid", B * g.d_model, &pb->resid));
  AIQ_TRY(ws(c, "pf.xn", B * g.d_model * (m.mlp_split ? 2 : 1), &pb->xn));
  AIQ_TRY(ws(c, "pf.qkv", B * nqkv, &pb->qkv));
  AIQ_TRY(ws(c, "pf.att", B * g.n_heads * g.head_dim, &pb->att));
  AIQ_TRY(ws(c, "pf.act", std::max(B, max_rows) * g.d_ffn * (m.mlp_split ? 2 : 1), &pb->act));
  AIQ_TRY(ws(c, "pf.resid_last", max_rows * g.d_model, &pb->resid_last));
  AIQ_TRY(ws(c, "pf.ss_attn", B * (g.d_model / 128), &pb->ss_attn));
  AIQ_TRY(ws(c, "pf.last_compact", max_rows, &pb->last_compact));
  return AIQ_OK;
}

// Decoder forward over one packed chunk of n_seqs sequences / T tokens.
// pkv_in (optional): per-layer keys/values [L][P][2 Hkv hd] of the shared
// prefix that every sequence attends; pkv_out (optional): where this pass
// stores its own keys/values per layer (the prefix pass).
// rows_only_last: the final layer's O-projection and MLP run only on each
// sequence's last token (the only position whose output reaches the label
// head); the result lands in b.resid_last, rows in sequence order.
aiq_status run_layers(aiq_ctx* c, ModelD& m, const PrefillBufs& b, int64_t T, int64_t n_seqs, const __half* pkv_in,
                      int P_in, __half* pkv_out, bool rows_only_last) {
  const aiq_model_config& g = m.cfg;
  const int d = g.d_model, hd = g.head_dim, Hq = g.n_heads, Hkv = g.n_kv_heads, f = g.d_ffn;
  const int nqkv = (Hq + 2 * Hkv) * hd;
  const int64_t ldkv = 2 * static_cast<int64_t>(Hkv) * hd;
  const int M = static_cast<int>(T);
  // The attention-side RMSNorm is fused: the embedding and every down
  // projection leave the residual times the next attention norm's gain in
  // b.xn as fp16, with the residual's partial sums of squares in ss_attn, and
  // the QKV GEMM scales each row by 1/RMS in its epilogue.  The gain is put on
  // the activation, not folded into the QKV weights: a rounded weight
  // perturbs every token alike, and over 32 layers that was the largest error
  // of the fp16 path against the fp64 oracle.  The MLP-side norm is a
  // standalone kernel: fusing it into the O-projection epilogue cost more
  // there than the kernel it removed.
  const int parts = d / 128;
  {
    // bf16 row in; fp32 residual, fp16 copy and the partial sums of squares out
    ProfScope p(c, "embed", 0, double(T) * d * 8.0 + double(T) * parts * 4.0);
    launch_embed(b.tok, T, m.embed, d, b.resid, b.xn, b.ss_attn, m.layers[0].attn_norm, c->d_err, c->stream);
    counted(c, T > 0);
  }
  for (int l = 0; l < g.n_layers; ++l) {
    const LayerD& L = m.layers[l];
    GemmEpilogue e1;
    e1.kind = EPI_ROPE_F16;
    e1.out = b.qkv;
    e1.ldo = nqkv;
    e1.positions = b.pos;
    e1.rope_cos = static_cast<const float*>(m.rope_cos.p);
    e1.rope_sin = static_cast<const float*>(m.rope_sin.p);
    e1.rope_cols = (Hq + Hkv) * hd;
    e1.head_dim = hd;
    e1.err = c->d_err;
    e1.row_ss = b.ss_attn;
    e1.ss_parts = parts;
    e1.d_norm = static_cast<float>(d);
    e1.eps = g.rms_eps;
    AIQ_TRY(gemm(c, "gemm_qkv_rope", b.xn, d, L.wqkv, d, M, nqkv, d, m.bn_qkv, e1));
    if (pkv_out && T > 0)
      CUDA_TRY(cudaMemcpy2DAsync(pkv_out + l * T * ldkv, ldkv * sizeof(__half), b.qkv + Hq * hd,
                                 nqkv * sizeof(__half), ldkv * sizeof(__half), T, cudaMemcpyDeviceToDevice, c->stream));
    AIQ_TRY(attention(c, b.qkv, T, n_seqs, b.seq_start, b.tile_seq, b.tile_q0, b.n_tiles, Hq, Hkv, hd,
                      pkv_in ? pkv_in + l * P_in * ldkv : nullptr, P_in, b.att));
    const bool prune = rows_only_last && l == g.n_layers - 1;
    GemmEpilogue e2;
    e2.kind = EPI_RESID_F32;
    e2.ldo = d;
    e2.err = c->d_err;
    e2.ss_parts = parts;
    GemmEpilogue e3;
    e3.kind = EPI_SWIGLU_F16;
    e3.out = b.act;
    e3.ldo = f;
    e3.err = c->d_err;
    // two-term MLP activations (m.mlp_split): rows of xn and act twice as wide
    const int ks = m.mlp_split ? 2 : 1;
    if (m.mlp_split) {
      e3.ldo = 2 * f;
      e3.lo_off = f;
    }
    if (!prune) {
      e2.out = b.resid;
      e2.kind = EPI_RESID_ADD;  // the residual add is done by the TMA unit (no fp16 copy wanted here)
      AIQ_TRY(gemm(c, "gemm_o_resid", b.att, Hq * hd, L.wo, Hq * hd, M, d, Hq * hd, m.bn_o, e2));
      e2.kind = EPI_RESID_F32;
      {
        ProfScope p(c, "rmsnorm", 0, 6.0 * double(T) * d);  // fp32 in, fp16 out
        launch_rmsnorm(b.resid, T, d, L.mlp_norm, g.rms_eps, b.xn, c->d_err, c->stream, m.mlp_split);
        counted(c, T > 0);
      }
      AIQ_TRY(gemm(c, "gemm_gateup_swiglu", b.xn, ks * d, L.wgu, ks * d, M, 2 * f, ks * d, m.bn_gu, e3, d));
      // the down projection's epilogue prepares the next layer's attention norm
      // (b.xn is free again: the gate/up GEMM before it has consumed it)
      e2.xh_out = b.xn;
      e2.xh_gain = l + 1 < g.n_layers ? m.layers[l + 1].attn_norm : nullptr;
      e2.ss_out = b.ss_attn;
      AIQ_TRY(gemm(c, "gemm_down_resid", b.act, ks * f, L.wd, ks * f, M, d, ks * f, m.bn_d, e2, f));
    } else {
      // final layer, rows only: gather each sequence's last token (the
      // attention output is dead afterwards, so its rows are packed into
      // b.qkv), then O-projection, RMSNorm and the MLP on those rows alone
      {
        ProfScope p(c, "gather_last", 0, 0);
        launch_gather_last(b.att, Hq * hd, b.resid, d, b.last_idx, n_seqs, b.qkv, b.resid_last, b.last_compact,
                           c->stream);
        counted(c, n_seqs > 0);
      }
      const int Mo = static_cast<int>(n_seqs);
      e2.out = b.resid_last;
      e2.kind = EPI_RESID_ADD;
      AIQ_TRY(gemm(c, "gemm_o_resid", b.qkv, Hq * hd, L.wo, Hq * hd, Mo, d, Hq * hd, m.bn_o, e2));
      {
        ProfScope p(c, "rmsnorm", 0, 6.0 * double(Mo) * d);
        launch_rmsnorm(b.resid_last, Mo, d, L.mlp_norm, g.rms_eps, b.xn, c->d_err, c->stream, m.mlp_split);
        counted(c, Mo > 0);
      }
      AIQ_TRY(gemm(c, "gemm_gateup_swiglu", b.xn, ks * d, L.wgu, ks * d, Mo, 2 * f, ks * d, m.bn_gu, e3, d));
      AIQ_TRY(gemm(c, "gemm_down_resid", b.act, ks * f, L.wd, ks * f, Mo, d, ks * f, m.bn_d, e2, f));
    }
  }
  return AIQ_OK;
}

struct QueryState {
  int64_t S = 0;
  int32_t* ids = nullptr;        // candidate (probe) rows; Q4 pairs: the A rows
  int32_t* ids2 = nullptr;       // Q4 pairs: the B rows (their text follows A's)
  int32_t* build_rows = nullptr; // joins
  float* logits = nullptr;       // [S, K]
  int64_t T = 0, n_chunks = 0, pairs = 0;  // T: row tokens (prefix excluded)
  int64_t P = 0;                            // prefix tokens, run once
};

// Generation state of an AI_TRANSFORM query (Table 1): greedy decoding of
// every candidate row after its chunk's prefill.
struct GenPlan {
  int max_new = 0, eos = -1, pad = 0;
  int32_t* tok = nullptr;  // [S, max_new] generated tokens (device)
  int32_t* len = nullptr;  // [S] tokens before the eos (device)
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> spans;  // decode time per chunk
  double flops = 0;
  int64_t steps = 0;
};

// Full-vocabulary LM head in the GEMM's operand format, made once per model.
aiq_status ensure_lm_f16(aiq_ctx* c, ModelD& m) {
  if (m.lm_f16) return AIQ_OK;
  const aiq_model_config& g = m.cfg;
  const int vpad = (g.vocab + 255) / 256 * 256;
  __half* w = nullptr;
  float* b = nullptr;
  void* p = nullptr;
  AIQ_TRY(dalloc(c, &p, static_cast<size_t>(vpad) * g.d_model * sizeof(__half)));
  w = static_cast<__half*>(p);
  m.allocs.push_back(DevBuf{p, std::max<size_t>(static_cast<size_t>(vpad) * g.d_model * sizeof(__half), 256)});
  AIQ_TRY(dalloc(c, &p, static_cast<size_t>(vpad) * sizeof(float)));
  b = static_cast<float*>(p);
  m.allocs.push_back(DevBuf{p, std::max<size_t>(static_cast<size_t>(vpad) * sizeof(float), 256)});
  CUDA_TRY(cudaMemsetAsync(w, 0, static_cast<size_t>(vpad) * g.d_model * sizeof(__half), c->stream));
  launch_bf16_to_f16(m.lm_head, w, g.vocab, g.d_model, 0, 0, c->d_err, c->stream);
  launch_bias_f32(m.lm_bias, g.vocab, vpad, b, c->stream);
  counted(c, 2);
  AIQ_TRY(sync_and_check(c));
  m.lm_f16 = w;
  m.lm_bias_f32 = b;
  m.vpad = vpad;
  return AIQ_OK;
}

struct DecodeBufs {
  __half *kvc, *gkv;  // [L][Tc][2 kd] prompt keys/values of the chunk; [L][R][gcap][2 kd] generated ones
  int gcap;
  unsigned long long* best;
  int32_t *done, *next, *pos;
};

// Greedy tokens of the LM head for R rows of normalised hidden states in b.xn.
aiq_status lm_argmax_select(aiq_ctx* c, ModelD& m, const PrefillBufs& b, const DecodeBufs& d, int R, int t,
                            GenPlan* gp, int64_t r0, int P) {
  GemmEpilogue e;
  e.kind = EPI_ARGMAX;
  e.bias = m.lm_bias_f32;
  e.best = d.best;
  e.err = c->d_err;
  AIQ_TRY(gemm(c, "gemm_lm_argmax", b.xn, m.cfg.d_model, m.lm_f16, m.cfg.d_model, R, m.vpad, m.cfg.d_model, 256, e));
  ProfScope p(c, "decode_select", 0, 0);
  launch_decode_select(d.best, R, t, gp->max_new, gp->eos, gp->pad, m.cfg.vocab, d.done,
                       gp->tok + r0 * gp->max_new, gp->len + r0, d.next, d.pos, b.seq_start, P, c->d_err, c->stream);
  counted(c, 1);
  return AIQ_OK;
}

// One decoder pass over R single-token rows (each row's newest token, at its
// own position), keys/values appended to generated slot `slot`.
aiq_status decode_layers(aiq_ctx* c, ModelD& m, const PrefillBufs& b, const DecodeBufs& d, int R, int64_t Tc,
                         const __half* pkv, int P, int slot) {
  const aiq_model_config& g = m.cfg;
  const int dm = g.d_model, hd = g.head_dim, Hq = g.n_heads, Hkv = g.n_kv_heads, f = g.d_ffn;
  const int nqkv = (Hq + 2 * Hkv) * hd;
  const int64_t ldkv = 2 * static_cast<int64_t>(Hkv) * hd;
  const int parts = dm / 128;
  {
    ProfScope p(c, "embed", 0, double(R) * dm * 8.0 + double(R) * parts * 4.0);
    launch_embed(d.next, R, m.embed, dm, b.resid, b.xn, b.ss_attn, m.layers[0].attn_norm, c->d_err, c->stream);
    counted(c, 1);
  }
  for (int l = 0; l < g.n_layers; ++l) {
    const LayerD& L = m.layers[l];
    GemmEpilogue e1;
    e1.kind = EPI_ROPE_F16;
    e1.out = b.qkv;
    e1.ldo = nqkv;
    e1.positions = d.pos;
    e1.rope_cos = static_cast<const float*>(m.rope_cos.p);
    e1.rope_sin = static_cast<const float*>(m.rope_sin.p);
    e1.rope_cols = (Hq + Hkv) * hd;
    e1.head_dim = hd;
    e1.err = c->d_err;
    e1.row_ss = b.ss_attn;
    e1.ss_parts = parts;
    e1.d_norm = static_cast<float>(dm);
    e1.eps = g.rms_eps;
    AIQ_TRY(gemm(c, "dec_gemm_qkv_rope", b.xn, dm, L.wqkv, dm, R, nqkv, dm, m.bn_qkv, e1));
    {
      // keys read per row: P + len + slot + 1; summed over the rows: R (P + slot + 1) + Tc
      const double keys = double(R) * (P + slot + 1) + double(Tc);
      ProfScope p(c, "decode_attention", 4.0 * Hq * hd * keys,
                  keys * ldkv * 2.0 + double(R) * (nqkv + Hq * hd + ldkv) * 2.0);
      const int e = launch_decode_attention(b.qkv, nqkv, R, Hq, Hkv, hd, pkv ? pkv + l * P * ldkv : nullptr, P,
                                            d.kvc + l * Tc * ldkv, b.seq_start,
                                            d.gkv + static_cast<int64_t>(l) * R * d.gcap * ldkv, d.gcap, slot, b.att,
                                            c->d_err, c->stream);
      counted(c, 1);
      if (e != 0)
        return fail(AIQ_ERR_CUDA, std::string("decode attention launch: ") +
                                      cudaGetErrorString(static_cast<cudaError_t>(e)));
    }
    GemmEpilogue e2;
    e2.kind = EPI_RESID_ADD;
    e2.out = b.resid;
    e2.ldo = dm;
    e2.err = c->d_err;
    e2.ss_parts = parts;
    AIQ_TRY(gemm(c, "dec_gemm_o_resid", b.att, Hq * hd, L.wo, Hq * hd, R, dm, Hq * hd, m.bn_o, e2));
    e2.kind = EPI_RESID_F32;
    {
      ProfScope p(c, "rmsnorm", 0, 6.0 * double(R) * dm);
      launch_rmsnorm(b.resid, R, dm, L.mlp_norm, g.rms_eps, b.xn, c->d_err, c->stream, m.mlp_split);
      counted(c, 1);
    }
    const int ks = m.mlp_split ? 2 : 1;
    GemmEpilogue e3;
    e3.kind = EPI_SWIGLU_F16;
    e3.out = b.act;
    e3.ldo = ks * f;
    e3.lo_off = m.mlp_split ? f : 0;
    e3.err = c->d_err;
    AIQ_TRY(gemm(c, "dec_gemm_gateup_swiglu", b.xn, ks * dm, L.wgu, ks * dm, R, 2 * f, ks * dm, m.bn_gu, e3, dm));
    e2.xh_out = b.xn;
    e2.xh_gain = l + 1 < g.n_layers ? m.layers[l + 1].attn_norm : nullptr;
    e2.ss_out = b.ss_attn;
    AIQ_TRY(gemm(c, "dec_gemm_down_resid", b.act, ks * f, L.wd, ks * f, R, dm, ks * f, m.bn_d, e2, f));
  }
  return AIQ_OK;
}

// max_new greedy steps for the R rows of one chunk whose prefill just ran
// (final hidden state of each row's last prompt token in b.resid_last).
aiq_status decode_chunk(aiq_ctx* c, ModelD& m, const PrefillBufs& b, const DecodeBufs& d, int R, int64_t Tc,
                        const __half* pkv, int P, const float* prefix_last, int64_t r0, GenPlan* gp) {
  const aiq_model_config& g = m.cfg;
  launch_patch_empty_rows(b.resid_last, b.last_compact, prefix_last, R, g.d_model, c->stream);
  {
    ProfScope p(c, "rmsnorm", 0, 6.0 * double(R) * g.d_model);
    launch_rmsnorm(b.resid_last, R, g.d_model, m.final_norm, g.rms_eps, b.xn, c->d_err, c->stream);
    counted(c, 2);
  }
  AIQ_TRY(lm_argmax_select(c, m, b, d, R, 0, gp, r0, P));
  for (int t = 1; t < gp->max_new; ++t) {
    AIQ_TRY(decode_layers(c, m, b, d, R, Tc, pkv, P, t - 1));
    {
      ProfScope p(c, "rmsnorm", 0, 6.0 * double(R) * g.d_model);
      launch_rmsnorm(b.resid, R, g.d_model, m.final_norm, g.rms_eps, b.xn, c->d_err, c->stream);
      counted(c, 1);
    }
    AIQ_TRY(lm_argmax_select(c, m, b, d, R, t, gp, r0, P));
  }
  // executed FLOPs: full LM head every step; decoder passes with attention over
  // P + len + t keys per row (sum over rows: R (P + t) + Tc)
  const double hq_hd = double(g.n_heads) * g.head_dim;
  gp->flops += double(gp->max_new) * 2.0 * g.d_model * m.vpad * R;
  for (int t = 1; t < gp->max_new; ++t)
    gp->flops += m.linear_flops_per_token * R + 4.0 * hq_hd * g.n_layers * (double(R) * (P + t) + double(Tc));
  gp->steps += gp->max_new;
  return AIQ_OK;
}

aiq_status prefill_phase(aiq_ctx* c, const TableD& t, ModelD& m, const aiq_select* q, QueryState* st,
                         GenPlan* gp = nullptr) {
  const ColD& col = t.cols[q->text_column];
  const int K = gp ? 0 : q->n_labels;
  const int64_t S = st->S;
  const int32_t P = q->prefix_len;
  float* logits = nullptr;
  if (!gp) {
    AIQ_TRY(ws(c, "q.logits", std::max<int64_t>(S * K, 1), &logits));
    st->logits = logits;
  }
  if (S == 0) return AIQ_OK;
  int32_t *lens, *prefix_d, *labels_d = nullptr;
  int64_t *cu, *scan_scratch;
  unsigned long long* pairs_d;
  AIQ_TRY(ws(c, "q.lens", S, &lens));
  AIQ_TRY(ws(c, "q.cu", S + 1, &cu));
  AIQ_TRY(ws(c, "q.scan", 2 * (S / kRowsPerBlock + 2), &scan_scratch));
  AIQ_TRY(ws(c, "q.pairs", 1, &pairs_d));
  AIQ_TRY(ws(c, "q.prefix", std::max<int32_t>(P, 1), &prefix_d));
  if (P > 0) CUDA_TRY(cudaMemcpyAsync(prefix_d, q->prefix, P * sizeof(int32_t), cudaMemcpyHostToDevice, c->stream));
  if (K > 0) {
    AIQ_TRY(ws(c, "q.labels", K, &labels_d));
    CUDA_TRY(cudaMemcpyAsync(labels_d, q->label_ids, K * sizeof(int32_t), cudaMemcpyHostToDevice, c->stream));
  }
  CUDA_TRY(cudaMemsetAsync(pairs_d, 0, sizeof(unsigned long long), c->stream));
  {
    ProfScope p(c, "pack_plan", 0, 0);
    launch_row_lengths(col.offsets, st->ids, S, P, lens, pairs_d, c->stream, st->ids2);
    launch_scan_lengths(lens, S, cu, scan_scratch, c->stream);
    counted(c, 4);
  }
  CUDA_TRY(cudaMemcpyAsync(c->h_pin + 1, pairs_d, sizeof(int64_t), cudaMemcpyDeviceToHost, c->stream));
  AIQ_TRY(read_i64(c, cu + S, 1, c->h_pin));
  const int64_t T = c->h_pin[0];
  st->T = T;
  st->pairs = c->h_pin[1];
  st->P = P;
  const int64_t max_len = col.max_len * (st->ids2 ? 2 : 1);  // longest row text; the prefix runs on its own
  int64_t n_chunks = 1, step = 0, rows_per_chunk = 0;
  if (gp) {
    // a chunk's rows decode together, one token each per step: as few chunks
    // of equal row counts as fit at most decode_rows rows, 2^20 tokens and
    // ~32 GB of prompt keys/values each (and of generated-token keys/values:
    // long generations decode fewer rows at a time).  (Splitting further to
    // fill the decode GEMMs' last tile wave measured slower: more launches.)
    const int64_t per_row = T / S + 1;
    const int64_t kv_row = 2 * int64_t(m.cfg.n_layers) * 2 * m.cfg.n_kv_heads * m.cfg.head_dim;  // bytes/token
    const int64_t kv_cap = (int64_t(32) << 30) / kv_row;
    const int64_t gen_rows_cap = std::max<int64_t>(1, (int64_t(32) << 30) / (kv_row * std::max(gp->max_new - 1, 1)));
    const int64_t row_cap = std::max<int64_t>(
        1, std::min<int64_t>({c->decode_rows, (int64_t(1) << 20) / per_row, kv_cap / per_row, gen_rows_cap}));
    n_chunks = (S + row_cap - 1) / row_cap;
    rows_per_chunk = (S + n_chunks - 1) / n_chunks;
  } else {
    const int64_t B = std::max<int64_t>(std::max<int64_t>(c->token_budget, max_len), P);
    step = B - max_len + 1;
    n_chunks = std::max<int64_t>(1, (T + step - 1) / step);
  }
  st->n_chunks = n_chunks;
  int64_t* chunk_d;
  AIQ_TRY(ws(c, "q.chunks", 2 * (n_chunks + 1), &chunk_d));
  if (gp)
    launch_chunk_bounds_rows(cu, S, rows_per_chunk, n_chunks, chunk_d, c->stream);
  else
    launch_chunk_bounds(cu, S, step, n_chunks, chunk_d, c->stream);
  counted(c, 1);
  std::vector<int64_t> chunks(2 * (n_chunks + 1));
  CUDA_TRY(cudaMemcpyAsync(chunks.data(), chunk_d, chunks.size() * sizeof(int64_t), cudaMemcpyDeviceToHost, c->stream));
  AIQ_TRY(sync_and_check(c));
  int64_t Bmax = P, Rmax = 1;
  for (int64_t i = 0; i < n_chunks; ++i) {
    Bmax = std::max(Bmax, chunks[2 * (i + 1) + 1] - chunks[2 * i + 1]);
    Rmax = std::max(Rmax, chunks[2 * (i + 1)] - chunks[2 * i]);
  }
  AIQ_TRY(ensure_rope(c, m, static_cast<int>(P + max_len + (gp ? gp->max_new : 0))));
  PrefillBufs pb;
  AIQ_TRY(prefill_bufs(c, m, std::max<int64_t>(Bmax, 64), Rmax, &pb));
  const aiq_model_config& g = m.cfg;
  const int64_t ldkv = 2 * static_cast<int64_t>(g.n_kv_heads) * g.head_dim;
  DecodeBufs db{};
  if (gp) {
    AIQ_TRY(ensure_lm_f16(c, m));
    db.gcap = std::max(gp->max_new - 1, 1);
    AIQ_TRY(ws(c, "g.kvc", static_cast<int64_t>(g.n_layers) * std::max<int64_t>(Bmax, 1) * ldkv, &db.kvc));
    AIQ_TRY(ws(c, "g.gkv", static_cast<int64_t>(g.n_layers) * Rmax * db.gcap * ldkv, &db.gkv));
    AIQ_TRY(ws(c, "g.best", Rmax, &db.best));
    AIQ_TRY(ws(c, "g.done", Rmax, &db.done));
    AIQ_TRY(ws(c, "g.next", Rmax, &db.next));
    AIQ_TRY(ws(c, "g.pos", Rmax, &db.pos));
    CUDA_TRY(cudaMemsetAsync(db.best, 0, Rmax * sizeof(unsigned long long), c->stream));
  }
  __half* pkv = nullptr;
  float* prefix_last;
  AIQ_TRY(ws(c, "pf.prefix_last", g.d_model, &prefix_last));
  if (P > 0) {
    // the shared prefix once: its per-layer keys/values and its last hidden state
    AIQ_TRY(ws(c, "pf.prefix_kv", static_cast<int64_t>(g.n_layers) * P * ldkv, &pkv));
    NvtxPhase pr("prefix");
    launch_pack_prefix(prefix_d, P, pb.tok, pb.pos, pb.seq_start, c->stream);
    counted(c, 1);
    AIQ_TRY(run_layers(c, m, pb, P, 1, nullptr, 0, pkv, false));
    CUDA_TRY(cudaMemcpyAsync(prefix_last, pb.resid + static_cast<int64_t>(P - 1) * g.d_model, g.d_model * sizeof(float),
                             cudaMemcpyDeviceToDevice, c->stream));
  }
  for (int64_t i = 0; i < n_chunks; ++i) {
    const int64_t r0 = chunks[2 * i], r1 = chunks[2 * (i + 1)];
    const int64_t Tc = chunks[2 * (i + 1) + 1] - chunks[2 * i + 1];
    if (r1 <= r0) continue;
    NvtxPhase chunk_range("chunk");
    {
      ProfScope p(c, "pack_chunk", 0, 0);
      launch_pack_chunk(cu, st->ids, col.offsets, static_cast<const int32_t*>(col.data), P, r0, r1, pb.tok, pb.pos,
                        pb.seq_start, pb.last_idx, c->stream, st->ids2);
      counted(c, 1);
    }
    // generation keeps every layer's prompt keys/values of the chunk for the decode steps
    AIQ_TRY(run_layers(c, m, pb, Tc, r1 - r0, pkv, static_cast<int>(P), gp ? db.kvc : nullptr, true));
    if (gp) {
      cudaEvent_t e0 = take_event(c), e1 = take_event(c);
      CUDA_TRY(cudaEventRecord(e0, c->stream));
      AIQ_TRY(decode_chunk(c, m, pb, db, static_cast<int>(r1 - r0), Tc, pkv, P, prefix_last, r0, gp));
      CUDA_TRY(cudaEventRecord(e1, c->stream));
      gp->spans.push_back({e0, e1});
    } else {
      ProfScope p(c, "label_head", 0, 0);
      launch_label_head(pb.resid_last, pb.last_compact, prefix_last, r1 - r0, g.d_model, m.final_norm, g.rms_eps,
                        m.lm_head, m.lm_bias, labels_d, K, logits + r0 * K, c->stream);
      counted(c, 1);
    }
  }
  return AIQ_OK;
}

// ------------------------------------------------------- aggregate phase ---

aiq_status aggregate_phase(aiq_ctx* c, const aiq_select* q, QueryState* st, const TableD* build, int32_t build_key,
                           ResultH& R, const TableD* probe = nullptr) {
  const int K = q->n_labels;
  const int64_t S = st->S;
  const int64_t nb = (S + kRowsPerBlock - 1) / kRowsPerBlock;
  int32_t *dec, *bcnt;
  uint32_t* ybits;
  int64_t* boff;
  unsigned long long* lcnt;
  AIQ_TRY(ws(c, "a.dec", std::max<int64_t>(S, 1), &dec));
  AIQ_TRY(ws(c, "a.bits", std::max<int64_t>(nb, 1) * (kRowsPerBlock / 32), &ybits));
  AIQ_TRY(ws(c, "a.bcnt", std::max<int64_t>(nb, 1), &bcnt));
  AIQ_TRY(ws(c, "a.boff", nb + 1, &boff));
  AIQ_TRY(ws(c, "a.lcnt", 16, &lcnt));
  CUDA_TRY(cudaMemsetAsync(lcnt, 0, 16 * sizeof(unsigned long long), c->stream));
  {
    ProfScope p(c, "decide", 0, 0);
    launch_decide(st->logits, S, K, dec, ybits, bcnt, lcnt, c->stream);
    counted(c, S > 0);
  }
  R.label_counts.resize(K);
  CUDA_TRY(cudaMemcpyAsync(R.label_counts.data(), lcnt, K * sizeof(int64_t), cudaMemcpyDeviceToHost, c->stream));
  if (q->agg == AIQ_AGG_ROW_IDS && K == 2 && S > 0) {
    launch_scan_counts(bcnt, nb, boff, c->stream);
    AIQ_TRY(read_i64(c, boff + nb, 1, c->h_pin));
    const int64_t Y = c->h_pin[0];
    int32_t *pos, *rows;
    AIQ_TRY(ws(c, "a.pos", std::max<int64_t>(Y, 1), &pos));
    AIQ_TRY(ws(c, "a.rows", std::max<int64_t>(Y, 1), &rows));
    launch_compact(ybits, boff, S, pos, st->ids, rows, c->stream);
    counted(c, 2);
    R.row_ids.resize(Y);
    if (Y) CUDA_TRY(cudaMemcpyAsync(R.row_ids.data(), rows, Y * sizeof(int32_t), cudaMemcpyDeviceToHost, c->stream));
    if (st->ids2) {  // Q4: the B row of every yes pair as well
      int32_t* rows_b;
      AIQ_TRY(ws(c, "a.rows_b", std::max<int64_t>(Y, 1), &rows_b));
      launch_gather_rows_i32(st->ids2, 1, pos, Y, rows_b, c->stream);
      counted(c, Y > 0);
      R.row_ids_b.resize(Y);
      if (Y)
        CUDA_TRY(cudaMemcpyAsync(R.row_ids_b.data(), rows_b, Y * sizeof(int32_t), cudaMemcpyDeviceToHost, c->stream));
    }
  }
  if (q->agg == AIQ_AGG_SUM && probe) {
    // Fig. 2: where(filter, values, 0).sum() over the candidates decided yes
    const ColD& col = probe->cols[q->sum_column];
    void *partial, *total;
    AIQ_TRY(ws(c, "a.sum_part", std::max<int64_t>(nb, 1) * 8, reinterpret_cast<uint8_t**>(&partial)));
    AIQ_TRY(ws(c, "a.sum", 8, reinterpret_cast<uint8_t**>(&total)));
    {
      ProfScope p(c, "masked_sum", 0, 0);
      launch_masked_sum(dec, st->ids, col.data, col.type, S, partial, total, c->stream);
      counted(c, 1 + (nb > 0));
    }
    R.sum_is_float = col.type == AIQ_FLOAT32;
    CUDA_TRY(cudaMemcpyAsync(&R.sum_bits, total, 8, cudaMemcpyDeviceToHost, c->stream));
  }
  if (q->agg == AIQ_AGG_GROUP_BUILD_KEY) {
    const int64_t nbr = build->n_rows;
    const int64_t gb = (nbr + kRowsPerBlock - 1) / kRowsPerBlock;
    unsigned long long* gcnt;
    uint32_t* gbits;
    int32_t* gbc;
    int64_t* goff;
    AIQ_TRY(ws(c, "g.cnt", std::max<int64_t>(nbr, 1), &gcnt));
    AIQ_TRY(ws(c, "g.bits", std::max<int64_t>(gb, 1) * (kRowsPerBlock / 32), &gbits));
    AIQ_TRY(ws(c, "g.bcnt", std::max<int64_t>(gb, 1), &gbc));
    AIQ_TRY(ws(c, "g.boff", gb + 1, &goff));
    CUDA_TRY(cudaMemsetAsync(gcnt, 0, std::max<int64_t>(nbr, 1) * sizeof(unsigned long long), c->stream));
    {
      ProfScope p(c, "group_by", 0, 0);
      launch_group_build(dec, st->build_rows, S, gcnt, c->stream);
      launch_nonzero_mask(gcnt, nbr, gbits, gbc, c->stream);
      launch_scan_counts(gbc, gb, goff, c->stream);
      counted(c, (S > 0) + (nbr > 0) + 1);
    }
    AIQ_TRY(read_i64(c, goff + gb, 1, c->h_pin));
    const int64_t G = c->h_pin[0];
    int32_t* grows;
    int64_t *gkeys, *gcounts;
    AIQ_TRY(ws(c, "g.rows", std::max<int64_t>(G, 1), &grows));
    AIQ_TRY(ws(c, "g.keys", std::max<int64_t>(G, 1), &gkeys));
    AIQ_TRY(ws(c, "g.counts", std::max<int64_t>(G, 1), &gcounts));
    launch_compact(gbits, goff, nbr, grows, nullptr, nullptr, c->stream);
    launch_gather_groups(grows, G, static_cast<const int64_t*>(build->cols[build_key].data), gcnt, gkeys, gcounts,
                         c->stream);
    counted(c, (nbr > 0) + (G > 0));
    R.group_rows.resize(G);
    R.group_keys.resize(G);
    R.group_counts.resize(G);
    if (G) {
      CUDA_TRY(cudaMemcpyAsync(R.group_rows.data(), grows, G * 4, cudaMemcpyDeviceToHost, c->stream));
      CUDA_TRY(cudaMemcpyAsync(R.group_keys.data(), gkeys, G * 8, cudaMemcpyDeviceToHost, c->stream));
      CUDA_TRY(cudaMemcpyAsync(R.group_counts.data(), gcounts, G * 8, cudaMemcpyDeviceToHost, c->stream));
    }
  }
  if (q->flags & AIQ_FLAG_LOGITS) {
    R.logits.resize(S * K);
    R.decisions.resize(S);
    if (S) {
      CUDA_TRY(cudaMemcpyAsync(R.logits.data(), st->logits, S * K * 4, cudaMemcpyDeviceToHost, c->stream));
      CUDA_TRY(cudaMemcpyAsync(R.decisions.data(), dec, S * 4, cudaMemcpyDeviceToHost, c->stream));
    }
  }
  return AIQ_OK;
}

void finish_view(ResultH& R, const QueryState& st, int64_t n_input, int K, int agg) {
  aiq_result_view& v = R.v;
  v.n_input_rows = n_input;
  v.n_candidates = st.S;
  v.n_tokens = st.T + st.P * st.S;
  v.n_prefill_tokens = st.S > 0 ? st.T + st.P : 0;
  v.n_chunks = st.n_chunks;
  v.count = (K == 2 && !R.label_counts.empty()) ? R.label_counts[0] : -1;
  v.row_ids = R.row_ids.empty() ? nullptr : R.row_ids.data();
  v.n_row_ids = static_cast<int64_t>(R.row_ids.size());
  v.group_build_rows = R.group_rows.empty() ? nullptr : R.group_rows.data();
  v.group_keys = R.group_keys.empty() ? nullptr : R.group_keys.data();
  v.group_counts = R.group_counts.empty() ? nullptr : R.group_counts.data();
  v.n_groups = static_cast<int64_t>(R.group_rows.size());
  v.label_counts = R.label_counts.empty() ? nullptr : R.label_counts.data();
  v.n_labels = static_cast<int32_t>(R.label_counts.size());
  v.cand_row_ids = R.cand_ids.empty() ? nullptr : R.cand_ids.data();
  v.cand_build_rows = R.cand_build.empty() ? nullptr : R.cand_build.data();
  v.label_logits = R.logits.empty() ? nullptr : R.logits.data();
  v.decisions = R.decisions.empty() ? nullptr : R.decisions.data();
  v.row_ids_b = R.row_ids_b.empty() ? nullptr : R.row_ids_b.data();
  v.sum_int = R.sum_is_float ? 0 : static_cast<int64_t>(R.sum_bits);
  v.sum_float = 0.0;
  if (R.sum_is_float) std::memcpy(&v.sum_float, &R.sum_bits, 8);
  v.gen_max_new = R.gen_max_new;
  v.n_gen_rows = static_cast<int64_t>(R.gen_ids.size());
  v.gen_row_ids = R.gen_ids.empty() ? nullptr : R.gen_ids.data();
  v.gen_tokens = R.gen_tok.empty() ? nullptr : R.gen_tok.data();
  v.gen_text_len = R.gen_len.empty() ? nullptr : R.gen_len.data();
  (void)agg;
}

// The prompt half of a query: text column, token ids, prefix, length limits.
aiq_status validate_prompt(const TableD& t, const ModelD* m, const aiq_select* q, int64_t extra_positions) {
  if (!m) return fail(AIQ_ERR_NOT_FOUND, "unknown model handle");
  if (q->text_column < 0 || q->text_column >= static_cast<int32_t>(t.cols.size()) ||
      t.cols[q->text_column].type != AIQ_TOKENS)
    return fail(AIQ_ERR_INVALID_ARG, "text_column must name a TOKENS column");
  const int V = m->cfg.vocab;
  if (t.cols[q->text_column].max_id >= V) return fail(AIQ_ERR_INVALID_ARG, "a row token id is >= vocab");
  if (q->prefix_len < 0 || (q->prefix_len > 0 && !q->prefix)) return fail(AIQ_ERR_INVALID_ARG, "bad prefix");
  for (int i = 0; i < q->prefix_len; ++i)
    if (q->prefix[i] < 0 || q->prefix[i] >= V) return fail(AIQ_ERR_INVALID_ARG, "prefix token id out of range");
  if (q->prefix_len == 0 && t.cols[q->text_column].min_len == 0)
    return fail(AIQ_ERR_INVALID_ARG, "a row with empty text needs a non-empty prefix (its prompt would be empty)");
  if (q->prefix_len + t.cols[q->text_column].max_len + extra_positions > (1 << 20))
    return fail(AIQ_ERR_UNSUPPORTED, "a prompt is longer than 2^20 tokens");
  return AIQ_OK;
}

aiq_status validate_select(aiq_ctx* c, const TableD& t, const ModelD* m, const aiq_select* q) {
  if (!q) return fail(AIQ_ERR_INVALID_ARG, "select is NULL");
  const bool rel_only = q->flags & AIQ_FLAG_RELATIONAL_ONLY;
  if (rel_only) return AIQ_OK;
  AIQ_TRY(validate_prompt(t, m, q, 0));
  const int V = m->cfg.vocab;
  if (q->n_labels < 2 || q->n_labels > 16 || !q->label_ids) return fail(AIQ_ERR_INVALID_ARG, "n_labels must be 2..16");
  for (int i = 0; i < q->n_labels; ++i)
    if (q->label_ids[i] < 0 || q->label_ids[i] >= V) return fail(AIQ_ERR_INVALID_ARG, "label id out of range");
  if (q->agg < AIQ_AGG_COUNT || q->agg > AIQ_AGG_SUM) return fail(AIQ_ERR_INVALID_ARG, "unknown agg");
  if (q->agg == AIQ_AGG_SUM) {
    if (q->n_labels != 2) return fail(AIQ_ERR_INVALID_ARG, "SUM needs exactly 2 labels (yes, no)");
    if (q->sum_column < 0 || q->sum_column >= static_cast<int32_t>(t.cols.size()) ||
        t.cols[q->sum_column].type == AIQ_TOKENS)
      return fail(AIQ_ERR_INVALID_ARG, "sum_column must name an INT32, INT64 or FLOAT32 column");
  }
  if ((q->agg == AIQ_AGG_COUNT || q->agg == AIQ_AGG_ROW_IDS) && q->n_labels != 2)
    return fail(AIQ_ERR_INVALID_ARG, "COUNT / ROW_IDS need exactly 2 labels (yes, no)");
  if (q->agg == AIQ_AGG_GROUP_BUILD_KEY && q->n_labels != 2)
    return fail(AIQ_ERR_INVALID_ARG, "GROUP_BUILD_KEY needs exactly 2 labels (yes, no)");
  (void)c;
  return AIQ_OK;
}

aiq_status run_query(aiq_ctx* c, const TableD* build, int32_t build_key, const aiq_pred* build_preds, int32_t n_bp,
                     const TableD& probe, int32_t probe_key, ModelD* m, const aiq_select* q, aiq_result_h* out) {
  AIQ_TRY(validate_select(c, probe, m, q));
  const bool rel_only = q->flags & AIQ_FLAG_RELATIONAL_ONLY;
  PredSet ps{};
  AIQ_TRY(make_pred_set(probe, q->preds, q->n_preds, &ps));
  if (!rel_only && q->agg == AIQ_AGG_GROUP_BUILD_KEY && !build)
    return fail(AIQ_ERR_INVALID_ARG, "GROUP_BUILD_KEY needs a join");

  c->launches = 0;
  cudaEvent_t ev[4];
  for (auto& e : ev) e = take_event(c);
  NvtxPhase whole(build ? "aiq_run_join_select" : "aiq_run_select");
  NvtxPhase phase("relational");
  CUDA_TRY(cudaEventRecord(ev[0], c->stream));
  QueryState st;
  ProbeSpec pr;
  if (build) {
    PredSet bps{};
    AIQ_TRY(make_pred_set(*build, build_preds, n_bp, &bps));
    int64_t Sb = 0;
    int32_t* bids;
    AIQ_TRY(filter_compact(c, *build, bps, ProbeSpec{}, "jb", &Sb, &bids, nullptr));
    int64_t cap = 64;
    while (cap < 2 * Sb) cap <<= 1;
    unsigned long long* tk;
    int32_t* tv;
    AIQ_TRY(ws(c, "j.keys", cap, &tk));
    AIQ_TRY(ws(c, "j.vals", cap, &tv));
    {
      ProfScope p(c, "hash_build", 0, 0);
      launch_fill_u64(tk, cap, 0x8000000000000000ull, c->stream);
      launch_hash_build(static_cast<const int64_t*>(build->cols[build_key].data), bids, Sb, tk, tv, cap, c->d_err,
                        c->stream);
      counted(c, 1 + (Sb > 0));
    }
    pr.keys = static_cast<const int64_t*>(probe.cols[probe_key].data);
    pr.table_keys = tk;
    pr.table_vals = tv;
    pr.capacity = cap;
  }
  AIQ_TRY(filter_compact(c, probe, ps, pr, "sel", &st.S, &st.ids, build ? &st.build_rows : nullptr));
  CUDA_TRY(cudaEventRecord(ev[1], c->stream));

  ResultH R;
  if (rel_only || (q->flags & AIQ_FLAG_LOGITS)) {
    R.cand_ids.resize(st.S);
    if (st.S) CUDA_TRY(cudaMemcpyAsync(R.cand_ids.data(), st.ids, st.S * 4, cudaMemcpyDeviceToHost, c->stream));
    if (build) {
      R.cand_build.resize(st.S);
      if (st.S)
        CUDA_TRY(cudaMemcpyAsync(R.cand_build.data(), st.build_rows, st.S * 4, cudaMemcpyDeviceToHost, c->stream));
    }
  }
  if (!rel_only) {
    phase.begin("prefill");
    AIQ_TRY(prefill_phase(c, probe, *m, q, &st));
    CUDA_TRY(cudaEventRecord(ev[2], c->stream));
    phase.begin("aggregate");
    AIQ_TRY(aggregate_phase(c, q, &st, build, build_key, R, &probe));
  } else {
    CUDA_TRY(cudaEventRecord(ev[2], c->stream));
  }
  CUDA_TRY(cudaEventRecord(ev[3], c->stream));
  phase.end();
  AIQ_TRY(sync_and_check(c));
  float t01 = 0, t12 = 0, t23 = 0, t03 = 0;
  cudaEventElapsedTime(&t01, ev[0], ev[1]);
  cudaEventElapsedTime(&t12, ev[1], ev[2]);
  cudaEventElapsedTime(&t23, ev[2], ev[3]);
  cudaEventElapsedTime(&t03, ev[0], ev[3]);
  for (auto& e : ev) c->ev_pool.push_back(e);
  collect_profile(c);
  const int K = rel_only ? 0 : q->n_labels;
  finish_view(R, st, probe.n_rows, K, q->agg);
  R.v.ms_relational = t01;
  R.v.ms_prefill = t12;
  R.v.ms_aggregate = t23;
  R.v.ms_total = t03;
  if (!rel_only && m) {
    const aiq_model_config& g = m->cfg;
    const double pre = st.S > 0 ? static_cast<double>(st.P) : 0.0;
    // final layer: Q/K/V for every token, O-projection and MLP for each row's last token only
    const double d = g.d_model, qd = double(g.n_heads) * g.head_dim, kd = double(g.n_kv_heads) * g.head_dim;
    const double per_layer = m->linear_flops_per_token / g.n_layers;
    const double tail = 2.0 * (qd * d + 3.0 * d * g.d_ffn);
    R.v.prefill_flops = per_layer * (g.n_layers - 1) * (static_cast<double>(st.T) + pre) +
                        2.0 * d * (qd + 2 * kd) * static_cast<double>(st.T) + tail * static_cast<double>(st.S) +
                        per_layer * pre +
                        4.0 * g.n_heads * g.head_dim * g.n_layers * (static_cast<double>(st.pairs) + pre * (pre + 1) / 2) +
                        2.0 * g.d_model * K * static_cast<double>(st.S);
  }
  ResultH& dst = new_result(c, out);
  dst = std::move(R);
  finish_view(dst, st, probe.n_rows, K, q->agg);
  dst.v.ms_relational = t01;
  dst.v.ms_prefill = t12;
  dst.v.ms_aggregate = t23;
  dst.v.ms_total = t03;
  if (!rel_only && m) dst.v.prefill_flops = R.v.prefill_flops;
  dst.v.n_launches = c->launches;
  return AIQ_OK;
}

// Table 2 Q3 / Q5: relational phase, prefill + greedy decoding per chunk,
// then the LIKE filter and the result arrays.
aiq_status run_transform(aiq_ctx* c, const TableD& t, ModelD* m, const aiq_select* q, const aiq_generate* gen,
                         aiq_result_h* out) {
  AIQ_TRY(validate_prompt(t, m, q, gen->max_new_tokens));
  const int V = m->cfg.vocab;
  if (gen->max_new_tokens < 1 || gen->max_new_tokens > 4096)
    return fail(AIQ_ERR_INVALID_ARG, "max_new_tokens must be 1..4096");
  if (gen->eos_id < -1 || gen->eos_id >= V) return fail(AIQ_ERR_INVALID_ARG, "eos_id must be -1 or a token id");
  if (gen->pad_id < 0 || gen->pad_id >= V) return fail(AIQ_ERR_INVALID_ARG, "pad_id must be a token id");
  const bool like = gen->like_tokens != nullptr;
  if (like && (gen->like_len < 0 || gen->like_len > 256)) return fail(AIQ_ERR_INVALID_ARG, "like_len must be 0..256");
  for (int i = 0; like && i < gen->like_len; ++i)
    if (gen->like_tokens[i] < 0 || gen->like_tokens[i] >= V)
      return fail(AIQ_ERR_INVALID_ARG, "LIKE pattern token id out of range");
  PredSet ps{};
  AIQ_TRY(make_pred_set(t, q->preds, q->n_preds, &ps));

  c->launches = 0;
  cudaEvent_t ev[4];
  for (auto& e : ev) e = take_event(c);
  NvtxPhase whole("aiq_run_transform");
  NvtxPhase phase("relational");
  CUDA_TRY(cudaEventRecord(ev[0], c->stream));
  QueryState st;
  AIQ_TRY(filter_compact(c, t, ps, ProbeSpec{}, "sel", &st.S, &st.ids, nullptr));
  CUDA_TRY(cudaEventRecord(ev[1], c->stream));
  phase.begin("prefill");
  const int64_t S = st.S;
  const int W = gen->max_new_tokens;
  GenPlan gp;
  gp.max_new = W;
  gp.eos = gen->eos_id;
  gp.pad = gen->pad_id;
  AIQ_TRY(ws(c, "g.tok", std::max<int64_t>(S * W, 1), &gp.tok));
  AIQ_TRY(ws(c, "g.len", std::max<int64_t>(S, 1), &gp.len));
  AIQ_TRY(prefill_phase(c, t, *m, q, &st, &gp));
  CUDA_TRY(cudaEventRecord(ev[2], c->stream));
  phase.begin("aggregate");

  ResultH R;
  R.gen_max_new = W;
  if (!like) {
    R.gen_ids.resize(S);
    R.gen_tok.resize(S * W);
    R.gen_len.resize(S);
    if (S) {
      CUDA_TRY(cudaMemcpyAsync(R.gen_ids.data(), st.ids, S * 4, cudaMemcpyDeviceToHost, c->stream));
      CUDA_TRY(cudaMemcpyAsync(R.gen_tok.data(), gp.tok, S * W * 4, cudaMemcpyDeviceToHost, c->stream));
      CUDA_TRY(cudaMemcpyAsync(R.gen_len.data(), gp.len, S * 4, cudaMemcpyDeviceToHost, c->stream));
    }
  } else if (S > 0) {
    // LIKE on the device; only the matches' ids (and, if asked, their tokens) come back
    const int64_t nb = (S + kRowsPerBlock - 1) / kRowsPerBlock;
    int32_t *pat, *match, *bcnt, *pos, *rows;
    uint32_t* bits;
    int64_t* boff;
    AIQ_TRY(ws(c, "g.like", std::max(gen->like_len, 1), &pat));
    AIQ_TRY(ws(c, "g.match", S, &match));
    AIQ_TRY(ws(c, "g.bits", nb * (kRowsPerBlock / 32), &bits));
    AIQ_TRY(ws(c, "g.bcnt", nb, &bcnt));
    AIQ_TRY(ws(c, "g.boff", nb + 1, &boff));
    if (gen->like_len > 0)
      CUDA_TRY(cudaMemcpyAsync(pat, gen->like_tokens, gen->like_len * 4, cudaMemcpyHostToDevice, c->stream));
    {
      ProfScope p(c, "like_match", 0, 0);
      launch_like_match(gp.tok, gp.len, S, W, pat, gen->like_len, match, c->stream);
      launch_flag_mask(match, S, bits, bcnt, c->stream);
      launch_scan_counts(bcnt, nb, boff, c->stream);
      counted(c, 3);
    }
    AIQ_TRY(read_i64(c, boff + nb, 1, c->h_pin));
    const int64_t Y = c->h_pin[0];
    AIQ_TRY(ws(c, "g.mpos", std::max<int64_t>(Y, 1), &pos));
    AIQ_TRY(ws(c, "g.mrows", std::max<int64_t>(Y, 1), &rows));
    launch_compact(bits, boff, S, pos, st.ids, rows, c->stream);
    counted(c, 1);
    R.row_ids.resize(Y);
    if (Y) CUDA_TRY(cudaMemcpyAsync(R.row_ids.data(), rows, Y * 4, cudaMemcpyDeviceToHost, c->stream));
    R.label_counts.clear();
    if ((gen->flags & AIQ_GEN_MATCH_TOKENS) && Y > 0) {
      int32_t *mtok, *mlen;
      AIQ_TRY(ws(c, "g.mtok", Y * W, &mtok));
      AIQ_TRY(ws(c, "g.mlen", Y, &mlen));
      launch_gather_rows_i32(gp.tok, W, pos, Y, mtok, c->stream);
      launch_gather_rows_i32(gp.len, 1, pos, Y, mlen, c->stream);
      counted(c, 2);
      R.gen_ids = R.row_ids;
      R.gen_tok.resize(Y * W);
      R.gen_len.resize(Y);
      CUDA_TRY(cudaMemcpyAsync(R.gen_tok.data(), mtok, Y * W * 4, cudaMemcpyDeviceToHost, c->stream));
      CUDA_TRY(cudaMemcpyAsync(R.gen_len.data(), mlen, Y * 4, cudaMemcpyDeviceToHost, c->stream));
    }
  }
  CUDA_TRY(cudaEventRecord(ev[3], c->stream));
  AIQ_TRY(sync_and_check(c));
  float t01 = 0, t12 = 0, t23 = 0, t03 = 0, tdec = 0;
  cudaEventElapsedTime(&t01, ev[0], ev[1]);
  cudaEventElapsedTime(&t12, ev[1], ev[2]);
  cudaEventElapsedTime(&t23, ev[2], ev[3]);
  cudaEventElapsedTime(&t03, ev[0], ev[3]);
  for (auto& e : ev) c->ev_pool.push_back(e);
  for (auto& sp : gp.spans) {
    float ms = 0;
    cudaEventElapsedTime(&ms, sp.first, sp.second);
    tdec += ms;
    c->ev_pool.push_back(sp.first);
    c->ev_pool.push_back(sp.second);
  }
  collect_profile(c);
  ResultH& dst = new_result(c, out);
  dst = std::move(R);
  finish_view(dst, st, t.n_rows, 0, -1);
  dst.v.count = like ? static_cast<int64_t>(dst.row_ids.size()) : -1;
  dst.v.ms_relational = t01;
  dst.v.ms_prefill = t12;
  dst.v.ms_aggregate = t23;
  dst.v.ms_total = t03;
  dst.v.ms_decode = tdec;
  dst.v.decode_flops = gp.flops;
  dst.v.n_decode_steps = gp.steps;
  {
    const aiq_model_config& g = m->cfg;
    const double pre = S > 0 ? static_cast<double>(st.P) : 0.0;
    const double d = g.d_model, qd = double(g.n_heads) * g.head_dim, kd = double(g.n_kv_heads) * g.head_dim;
    const double per_layer = m->linear_flops_per_token / g.n_layers;
    const double tail = 2.0 * (qd * d + 3.0 * d * g.d_ffn);
    dst.v.prefill_flops = per_layer * (g.n_layers - 1) * (static_cast<double>(st.T) + pre) +
                          2.0 * d * (qd + 2 * kd) * static_cast<double>(st.T) + tail * static_cast<double>(S) +
                          per_layer * pre +
                          4.0 * g.n_heads * g.head_dim * g.n_layers * (static_cast<double>(st.pairs) + pre * (pre + 1) / 2);
  }
  dst.v.n_launches = c->launches;
  return AIQ_OK;
}

// Table 2 Q4: WHERE on the table, the key self-join into (a, b) pairs on the
// device, then AI_IF on every pair's prompt and the aggregate over pairs.
aiq_status run_pair_select(aiq_ctx* c, const TableD& t, int32_t key_col, ModelD* m, const aiq_select* q,
                           aiq_result_h* out) {
  if (q->flags & AIQ_FLAG_RELATIONAL_ONLY) return fail(AIQ_ERR_INVALID_ARG, "pair queries need the language model");
  AIQ_TRY(validate_select(c, t, m, q));
  AIQ_TRY(validate_prompt(t, m, q, t.cols[q->text_column].max_len));  // two texts per prompt
  if (q->n_labels != 2) return fail(AIQ_ERR_INVALID_ARG, "pair queries need exactly 2 labels (yes, no)");
  if (q->agg != AIQ_AGG_COUNT && q->agg != AIQ_AGG_ROW_IDS)
    return fail(AIQ_ERR_INVALID_ARG, "pair queries aggregate with COUNT or ROW_IDS");
  PredSet ps{};
  AIQ_TRY(make_pred_set(t, q->preds, q->n_preds, &ps));

  c->launches = 0;
  cudaEvent_t ev[4];
  for (auto& e : ev) e = take_event(c);
  NvtxPhase whole("aiq_run_pair_select");
  NvtxPhase phase("relational");
  CUDA_TRY(cudaEventRecord(ev[0], c->stream));
  int64_t S = 0;
  int32_t* ids;
  AIQ_TRY(filter_compact(c, t, ps, ProbeSpec{}, "sel", &S, &ids, nullptr));
  // self-join on the key: stable radix sort of the candidates' keys, pair offsets, pairs
  const int64_t tiles = (S + kRowsPerBlock - 1) / kRowsPerBlock;
  const int64_t n1 = std::max<int64_t>(S, 1);
  SelfJoinScratch w{};
  AIQ_TRY(ws(c, "p.keys", n1, &w.keys));
  AIQ_TRY(ws(c, "p.keys_tmp", n1, &w.keys_tmp));
  AIQ_TRY(ws(c, "p.vals", n1, &w.vals));
  AIQ_TRY(ws(c, "p.vals_tmp", n1, &w.vals_tmp));
  AIQ_TRY(ws(c, "p.heads", n1, &w.heads));
  AIQ_TRY(ws(c, "p.counts", n1, &w.counts));
  AIQ_TRY(ws(c, "p.head_excl", S + 1, &w.head_excl));
  AIQ_TRY(ws(c, "p.pair_off", S + 1, &w.pair_off));
  AIQ_TRY(ws(c, "p.group_start", S + 1, &w.group_start));
  AIQ_TRY(ws(c, "p.hist", 256 * std::max<int64_t>(tiles, 1), &w.hist));
  AIQ_TRY(ws(c, "p.hist_off", 256 * std::max<int64_t>(tiles, 1) + 1, &w.hist_off));
  const int64_t scan_n = std::max<int64_t>(S, 256 * tiles);
  AIQ_TRY(ws(c, "p.scan", 2 * ((scan_n + kRowsPerBlock - 1) / kRowsPerBlock + 1), &w.scan_tmp));
  {
    ProfScope p(c, "self_join", 0, 0);
    launch_self_join_pairs_plan(static_cast<const int64_t*>(t.cols[key_col].data), ids, S, w, c->stream);
    counted(c, S > 0 ? 1 + 8 * 5 + 3 + 3 + 3 : 0);
  }
  int64_t n_pairs = 0;
  if (S > 0) {
    AIQ_TRY(read_i64(c, w.pair_off + S, 1, c->h_pin));
    n_pairs = c->h_pin[0];
  }
  if (n_pairs > INT32_MAX) return fail(AIQ_ERR_CAPACITY, "more than 2^31 - 1 pairs");
  QueryState st;
  st.S = n_pairs;
  AIQ_TRY(ws(c, "p.a", std::max<int64_t>(n_pairs, 1), &st.ids));
  AIQ_TRY(ws(c, "p.b", std::max<int64_t>(n_pairs, 1), &st.ids2));
  launch_self_join_pairs_emit(ids, S, w, st.ids, st.ids2, c->stream);
  counted(c, S > 0);
  CUDA_TRY(cudaEventRecord(ev[1], c->stream));

  ResultH R;
  if (q->flags & AIQ_FLAG_LOGITS) {
    R.cand_ids.resize(n_pairs);
    R.cand_build.resize(n_pairs);
    if (n_pairs) {
      CUDA_TRY(cudaMemcpyAsync(R.cand_ids.data(), st.ids, n_pairs * 4, cudaMemcpyDeviceToHost, c->stream));
      CUDA_TRY(cudaMemcpyAsync(R.cand_build.data(), st.ids2, n_pairs * 4, cudaMemcpyDeviceToHost, c->stream));
    }
  }
  phase.begin("prefill");
  AIQ_TRY(prefill_phase(c, t, *m, q, &st));
  CUDA_TRY(cudaEventRecord(ev[2], c->stream));
  phase.begin("aggregate");
  AIQ_TRY(aggregate_phase(c, q, &st, nullptr, -1, R));
  CUDA_TRY(cudaEventRecord(ev[3], c->stream));
  phase.end();
  AIQ_TRY(sync_and_check(c));
  float t01 = 0, t12 = 0, t23 = 0, t03 = 0;
  cudaEventElapsedTime(&t01, ev[0], ev[1]);
  cudaEventElapsedTime(&t12, ev[1], ev[2]);
  cudaEventElapsedTime(&t23, ev[2], ev[3]);
  cudaEventElapsedTime(&t03, ev[0], ev[3]);
  for (auto& e : ev) c->ev_pool.push_back(e);
  collect_profile(c);
  ResultH& dst = new_result(c, out);
  dst = std::move(R);
  finish_view(dst, st, t.n_rows, 2, q->agg);
  dst.v.ms_relational = t01;
  dst.v.ms_prefill = t12;
  dst.v.ms_aggregate = t23;
  dst.v.ms_total = t03;
  {
    const aiq_model_config& g = m->cfg;
    const double pre = st.S > 0 ? static_cast<double>(st.P) : 0.0;
    const double d = g.d_model, qd = double(g.n_heads) * g.head_dim, kd = double(g.n_kv_heads) * g.head_dim;
    const double per_layer = m->linear_flops_per_token / g.n_layers;
    const double tail = 2.0 * (qd * d + 3.0 * d * g.d_ffn);
    dst.v.prefill_flops = per_layer * (g.n_layers - 1) * (static_cast<double>(st.T) + pre) +
                          2.0 * d * (qd + 2 * kd) * static_cast<double>(st.T) + tail * static_cast<double>(st.S) +
                          per_layer * pre +
                          4.0 * g.n_heads * g.head_dim * g.n_layers * (static_cast<double>(st.pairs) + pre * (pre + 1) / 2) +
                          2.0 * g.d_model * 2 * static_cast<double>(st.S);
  }
  dst.v.n_launches = c->launches;
  return AIQ_OK;
}

void free_model(aiq_ctx* c, ModelD& m) {
  for (auto& b : m.allocs) dfree(c, b.p, b.bytes);
  m.allocs.clear();
  dfree(c, m.rope_cos.p, m.rope_cos.bytes);
  dfree(c, m.rope_sin.p, m.rope_sin.bytes);
}

void free_table(aiq_ctx* c, TableD& t) {
  cudaStreamSynchronize(c->stream);  // uploads into these buffers may still be in flight
  for (auto& col : t.cols) {
    dfree(c, col.data, col.bytes);
    if (col.offsets) dfree(c, col.offsets, (t.n_rows + 1) * sizeof(int64_t));
  }
  t.cols.clear();
}

template <typename T>
aiq_status model_alloc(aiq_ctx* c, ModelD& m, size_t count, T** out) {
  void* p = nullptr;
  AIQ_TRY(dalloc(c, &p, count * sizeof(T)));
  m.allocs.push_back(DevBuf{p, std::max<size_t>(count * sizeof(T), 256)});
  *out = static_cast<T*>(p);
  return AIQ_OK;
}

int pick_bn(int n) { return n % 256 == 0 ? 256 : 128; }

}  // namespace

// =================================================================== C-ABI

extern "C" {

aiq_status aiq_init(int device, aiq_ctx** out) {
  if (!out) return fail(AIQ_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  int n = 0;
  CUDA_TRY(cudaGetDeviceCount(&n));
  if (device < 0 || device >= n) return fail(AIQ_ERR_INVALID_ARG, "no such CUDA device");
  CUDA_TRY(cudaSetDevice(device));
  cudaDeviceProp prop;
  CUDA_TRY(cudaGetDeviceProperties(&prop, device));
  if (prop.major != 10 || prop.minor != 3)
    return fail(AIQ_ERR_UNSUPPORTED, "this library is built for sm_103 (GB300) only");
  aiq_ctx* c = new aiq_ctx();
  c->device = device;
  c->num_sms = prop.multiProcessorCount;
  if (const char* cap = std::getenv("AIQ_DEVICE_BYTES_MAX")) c->bytes_max = std::strtoull(cap, nullptr, 10);
  cudaError_t e = cudaStreamCreateWithFlags(&c->stream, cudaStreamNonBlocking);
  if (e == cudaSuccess) e = cudaMalloc(&c->d_err, sizeof(int));
  if (e == cudaSuccess) e = cudaMemsetAsync(c->d_err, 0, sizeof(int), c->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
  if (e == cudaSuccess) e = cudaMallocHost(&c->h_pin, 64 * sizeof(int64_t));
  if (e != cudaSuccess) {
    cudaGetLastError();
    if (c->h_pin) cudaFreeHost(c->h_pin);
    if (c->d_err) cudaFree(c->d_err);
    if (c->stream) cudaStreamDestroy(c->stream);
    delete c;
    return fail(AIQ_ERR_CUDA, std::string("context setup: ") + cudaGetErrorString(e));
  }
  *out = c;
  g_err.clear();
  return AIQ_OK;
}

void aiq_shutdown(aiq_ctx* c) {
  if (!c) return;
  cudaSetDevice(c->device);
  cudaStreamSynchronize(c->stream);
  for (auto& kv : c->tables) free_table(c, kv.second);
  for (auto& kv : c->models) free_model(c, kv.second);
  for (auto& kv : c->ws) dfree(c, kv.second.p, kv.second.bytes);
  for (auto& r : c->prof) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  for (auto e : c->ev_pool) cudaEventDestroy(e);
  cudaFree(c->d_err);
  cudaFreeHost(c->h_pin);
  cudaStreamDestroy(c->stream);
  delete c;
}

aiq_status aiq_load_table(aiq_ctx* c, const aiq_column* cols, int32_t n_cols, int64_t n_rows, aiq_table* out) {
  if (!c || !out) return fail(AIQ_ERR_INVALID_ARG, "ctx/out is NULL");
  if (n_cols <= 0 || !cols) return fail(AIQ_ERR_INVALID_ARG, "no columns");
  if (n_rows < 0 || n_rows >= (int64_t(1) << 31)) return fail(AIQ_ERR_INVALID_ARG, "n_rows must be in [0, 2^31)");
  CUDA_TRY(cudaSetDevice(c->device));
  TableD t;
  t.n_rows = n_rows;
  for (int i = 0; i < n_cols; ++i) {
    const aiq_column& a = cols[i];
    ColD col;
    col.name = a.name ? a.name : "";
    col.type = a.type;
    if (a.type < AIQ_INT32 || a.type > AIQ_TOKENS) {
      free_table(c, t);
      return fail(AIQ_ERR_INVALID_ARG, "unknown column type");
    }
    if (!a.data && n_rows > 0) {
      free_table(c, t);
      return fail(AIQ_ERR_INVALID_ARG, "column data is NULL");
    }
    size_t bytes = 0;
    if (a.type == AIQ_TOKENS) {
      if (!a.offsets) {
        free_table(c, t);
        return fail(AIQ_ERR_INVALID_ARG, "TOKENS column without offsets");
      }
      if (a.offsets[0] != 0) {
        free_table(c, t);
        return fail(AIQ_ERR_INVALID_ARG, "token offsets must start at 0");
      }
      col.min_len = n_rows > 0 ? INT64_MAX : 0;
      for (int64_t r = 0; r < n_rows; ++r) {
        const int64_t len = a.offsets[r + 1] - a.offsets[r];
        if (len < 0) {
          free_table(c, t);
          return fail(AIQ_ERR_INVALID_ARG, "token offsets must be non-decreasing");
        }
        col.max_len = std::max(col.max_len, len);
        col.min_len = std::min(col.min_len, len);
      }
      const int64_t ntok = a.offsets[n_rows];
      if (ntok >= (int64_t(1) << 31)) {
        free_table(c, t);
        return fail(AIQ_ERR_UNSUPPORTED, "more than 2^31 tokens in one column");
      }
      const int32_t* ids = static_cast<const int32_t*>(a.data);
      for (int64_t k = 0; k < ntok; ++k) {
        if (ids[k] < 0) {
          free_table(c, t);
          return fail(AIQ_ERR_INVALID_ARG, "negative token id");
        }
        col.max_id = std::max<int64_t>(col.max_id, ids[k]);
      }
      bytes = static_cast<size_t>(ntok) * sizeof(int32_t);
      aiq_status st = dalloc(c, reinterpret_cast<void**>(&col.offsets), (n_rows + 1) * sizeof(int64_t));
      if (st != AIQ_OK) {
        free_table(c, t);
        return st;
      }
      const cudaError_t ce =
          cudaMemcpyAsync(col.offsets, a.offsets, (n_rows + 1) * sizeof(int64_t), cudaMemcpyHostToDevice, c->stream);
      if (ce != cudaSuccess) {
        cudaGetLastError();
        cudaStreamSynchronize(c->stream);
        dfree(c, col.offsets, (n_rows + 1) * sizeof(int64_t));
        free_table(c, t);
        return fail(AIQ_ERR_CUDA, std::string("table upload: ") + cudaGetErrorString(ce));
      }
    } else {
      bytes = static_cast<size_t>(n_rows) * (a.type == AIQ_INT64 ? 8 : 4);
    }
    col.bytes = bytes;
    aiq_status st = dalloc(c, &col.data, bytes);
    if (st != AIQ_OK) {
      cudaStreamSynchronize(c->stream);
      if (col.offsets) dfree(c, col.offsets, (n_rows + 1) * sizeof(int64_t));
      free_table(c, t);
      return st;
    }
    // on the context's stream: the query kernels that read the column run
    // there, and a copy on the legacy stream from pageable memory may still
    // be in flight when it returns
    const cudaError_t ce = bytes ? cudaMemcpyAsync(col.data, a.data, bytes, cudaMemcpyHostToDevice, c->stream)
                                 : cudaSuccess;
    t.cols.push_back(col);
    if (ce != cudaSuccess) {
      cudaGetLastError();
      free_table(c, t);
      return fail(AIQ_ERR_CUDA, std::string("table upload: ") + cudaGetErrorString(ce));
    }
  }
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    free_table(c, t);
    return fail(AIQ_ERR_CUDA, std::string("table upload: ") + cudaGetErrorString(e));
  }
  const int64_t h = c->next_handle++;
  c->tables[h] = std::move(t);
  *out = h;
  return AIQ_OK;
}

aiq_status aiq_free_table(aiq_ctx* c, aiq_table h) {
  if (!c) return fail(AIQ_ERR_INVALID_ARG, "ctx is NULL");
  auto it = c->tables.find(h);
  if (it == c->tables.end()) return fail(AIQ_ERR_NOT_FOUND, "unknown table handle");
  cudaStreamSynchronize(c->stream);
  free_table(c, it->second);
  c->tables.erase(it);
  return AIQ_OK;
}

aiq_status aiq_load_model(aiq_ctx* c, const aiq_model_config* cfg, const void* const* tensors, int32_t n_tensors,
                          aiq_model* out) {
  if (!c || !cfg || !tensors || !out) return fail(AIQ_ERR_INVALID_ARG, "NULL argument");
  const aiq_model_config g = *cfg;
  if (g.n_layers < 1 || g.d_model <= 0 || g.n_heads <= 0 || g.n_kv_heads <= 0 || g.d_ffn <= 0 || g.vocab <= 0)
    return fail(AIQ_ERR_INVALID_ARG, "model dimensions must be positive");
  if (g.n_heads % g.n_kv_heads) return fail(AIQ_ERR_INVALID_ARG, "n_heads must be a multiple of n_kv_heads");
  if (!(g.head_dim == 32 || g.head_dim == 64 || g.head_dim == 128))
    return fail(AIQ_ERR_UNSUPPORTED, "head_dim must be 32, 64 or 128");
  const int qd = g.n_heads * g.head_dim, kd = g.n_kv_heads * g.head_dim;
  if (g.d_model % 128 || g.d_ffn % 128 || qd % 128 || (qd + 2 * kd) % 128)
    return fail(AIQ_ERR_UNSUPPORTED, "d_model, d_ffn, Hq*hd and (Hq+2Hkv)*hd must be multiples of 128");
  if (n_tensors != 1 + 9 * g.n_layers + 3) return fail(AIQ_ERR_INVALID_ARG, "n_tensors must be 1 + 9 L + 3");
  for (int i = 0; i < n_tensors; ++i)
    if (!tensors[i]) return fail(AIQ_ERR_INVALID_ARG, "a tensor pointer is NULL");
  CUDA_TRY(cudaSetDevice(c->device));
  const int64_t d = g.d_model, f = g.d_ffn, V = g.vocab;
  ModelD m;
  m.cfg = g;
  m.mlp_split = c->mlp_split < 0 ? (g.n_layers >= 32 && g.d_model >= 4096) : c->mlp_split != 0;
  m.bn_qkv = pick_bn(qd + 2 * kd);
  m.bn_o = pick_bn(g.d_model);
  m.bn_gu = pick_bn(2 * g.d_ffn);
  m.bn_d = pick_bn(g.d_model);
  if (m.bn_qkv % g.head_dim) m.bn_qkv = 128;
  m.linear_flops_per_token = 2.0 * g.n_layers * (double(d) * (qd + 2 * kd) + double(qd) * d + 3.0 * d * f);
  auto up_bf16 = [&](const void* src, size_t count, uint16_t** dst) -> aiq_status {
    AIQ_TRY(model_alloc(c, m, count, dst));
    CUDA_TRY(cudaMemcpyAsync(*dst, src, count * 2, cudaMemcpyHostToDevice, c->stream));
    return AIQ_OK;
  };
  // bf16 weights into the staging buffer, ordered on the context's stream
  // before the conversion kernels that read them
  auto to_stage = [&](uint16_t* dst, const void* src, size_t count) -> aiq_status {
    CUDA_TRY(cudaMemcpyAsync(dst, src, count * 2, cudaMemcpyHostToDevice, c->stream));
    return AIQ_OK;
  };
  uint16_t* stage = nullptr;
  const size_t stage_elems = std::max<size_t>(2 * f * d, (size_t)(qd + 2 * kd) * d);
  void* sp = nullptr;
  aiq_status st = dalloc(c, &sp, stage_elems * 2);
  if (st != AIQ_OK) return st;
  stage = static_cast<uint16_t*>(sp);
  auto fail_model = [&](aiq_status s2) {
    cudaStreamSynchronize(c->stream);
    dfree(c, sp, stage_elems * 2);
    free_model(c, m);
    return s2;
  };
#define M_TRY(x)                           \
  do {                                     \
    aiq_status s_ = (x);                   \
    if (s_ != AIQ_OK) return fail_model(s_); \
  } while (0)
  int ti = 0;
  M_TRY(up_bf16(tensors[ti++], V * d, &m.embed));
  m.layers.resize(g.n_layers);
  for (int l = 0; l < g.n_layers; ++l) {
    LayerD& L = m.layers[l];
    M_TRY(up_bf16(tensors[ti++], d, &L.attn_norm));
    // q, k, v stacked then converted: [(Hq + 2 Hkv) hd, d] (exact: bf16 values in fp16)
    cudaStreamSynchronize(c->stream);
    M_TRY(to_stage(stage, tensors[ti++], size_t(qd) * d));
    M_TRY(to_stage(stage + size_t(qd) * d, tensors[ti++], size_t(kd) * d));
    M_TRY(to_stage(stage + size_t(qd + kd) * d, tensors[ti++], size_t(kd) * d));
    M_TRY(model_alloc(c, m, size_t(qd + 2 * kd) * d, &L.wqkv));
    launch_bf16_to_f16(stage, L.wqkv, qd + 2 * kd, d, 0, 0, c->d_err, c->stream);
    cudaStreamSynchronize(c->stream);
    M_TRY(to_stage(stage, tensors[ti++], size_t(d) * qd));
    M_TRY(model_alloc(c, m, size_t(d) * qd, &L.wo));
    launch_bf16_to_f16(stage, L.wo, d, qd, 0, 0, c->d_err, c->stream);
    M_TRY(up_bf16(tensors[ti++], d, &L.mlp_norm));
    cudaStreamSynchronize(c->stream);
    M_TRY(to_stage(stage, tensors[ti++], size_t(f) * d));
    M_TRY(to_stage(stage + size_t(f) * d, tensors[ti++], size_t(f) * d));
    // with mlp_split each weight row is stored twice along K ([W | W]), the
    // second copy multiplying the activation's low-order fp16 term
    const int ks = m.mlp_split ? 2 : 1;
    M_TRY(model_alloc(c, m, size_t(2 * f) * d * ks, &L.wgu));
    for (int k = 0; k < ks; ++k)
      launch_bf16_to_f16(stage, L.wgu + size_t(k) * d, 2 * f, d, m.bn_gu / 2, f, c->d_err, c->stream, ks * d);
    cudaStreamSynchronize(c->stream);
    M_TRY(to_stage(stage, tensors[ti++], size_t(d) * f));
    M_TRY(model_alloc(c, m, size_t(d) * f * ks, &L.wd));
    for (int k = 0; k < ks; ++k)
      launch_bf16_to_f16(stage, L.wd + size_t(k) * f, d, f, 0, 0, c->d_err, c->stream, ks * f);
  }
  M_TRY(up_bf16(tensors[ti++], d, &m.final_norm));
  M_TRY(up_bf16(tensors[ti++], V * d, &m.lm_head));
  M_TRY(up_bf16(tensors[ti++], V, &m.lm_bias));
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return fail_model(fail(AIQ_ERR_CUDA, std::string("model upload: ") + cudaGetErrorString(e)));
  int err = 0;
  cudaMemcpy(&err, c->d_err, sizeof(int), cudaMemcpyDeviceToHost);
  if (err) {
    cudaMemsetAsync(c->d_err, 0, sizeof(int), c->stream);
    return fail_model(fail(AIQ_ERR_UNSUPPORTED, "a linear weight is outside the fp16 range"));
  }
#undef M_TRY
  dfree(c, sp, stage_elems * 2);
  const int64_t h = c->next_handle++;
  c->models[h] = std::move(m);
  *out = h;
  return AIQ_OK;
}

aiq_status aiq_free_model(aiq_ctx* c, aiq_model h) {
  if (!c) return fail(AIQ_ERR_INVALID_ARG, "ctx is NULL");
  auto it = c->models.find(h);
  if (it == c->models.end()) return fail(AIQ_ERR_NOT_FOUND, "unknown model handle");
  cudaStreamSynchronize(c->stream);
  free_model(c, it->second);
  c->models.erase(it);
  return AIQ_OK;
}

aiq_status aiq_run_select(aiq_ctx* c, aiq_table table, aiq_model model, const aiq_select* q, aiq_result_h* out) {
  if (!c || !q || !out) return fail(AIQ_ERR_INVALID_ARG, "NULL argument");
  auto t = c->tables.find(table);
  if (t == c->tables.end()) return fail(AIQ_ERR_NOT_FOUND, "unknown table handle");
  ModelD* m = nullptr;
  auto mi = c->models.find(model);
  if (mi != c->models.end()) m = &mi->second;
  if (q->agg == AIQ_AGG_GROUP_BUILD_KEY && !(q->flags & AIQ_FLAG_RELATIONAL_ONLY))
    return fail(AIQ_ERR_INVALID_ARG, "GROUP_BUILD_KEY needs aiq_run_join_select");
  CUDA_TRY(cudaSetDevice(c->device));
  return run_query(c, nullptr, -1, nullptr, 0, t->second, -1, m, q, out);
}

aiq_status aiq_run_join_select(aiq_ctx* c, aiq_table build, int32_t build_key, const aiq_pred* build_preds,
                               int32_t n_build_preds, aiq_table probe, int32_t probe_key, aiq_model model,
                               const aiq_select* q, aiq_result_h* out) {
  if (!c || !q || !out) return fail(AIQ_ERR_INVALID_ARG, "NULL argument");
  auto b = c->tables.find(build);
  auto p = c->tables.find(probe);
  if (b == c->tables.end() || p == c->tables.end()) return fail(AIQ_ERR_NOT_FOUND, "unknown table handle");
  if (build_key < 0 || build_key >= static_cast<int32_t>(b->second.cols.size()) ||
      b->second.cols[build_key].type != AIQ_INT64)
    return fail(AIQ_ERR_INVALID_ARG, "build key must be an INT64 column");
  if (probe_key < 0 || probe_key >= static_cast<int32_t>(p->second.cols.size()) ||
      p->second.cols[probe_key].type != AIQ_INT64)
    return fail(AIQ_ERR_INVALID_ARG, "probe key must be an INT64 column");
  ModelD* m = nullptr;
  auto mi = c->models.find(model);
  if (mi != c->models.end()) m = &mi->second;
  CUDA_TRY(cudaSetDevice(c->device));
  return run_query(c, &b->second, build_key, build_preds, n_build_preds, p->second, probe_key, m, q, out);
}

aiq_status aiq_run_transform(aiq_ctx* c, aiq_table table, aiq_model model, const aiq_select* q,
                             const aiq_generate* gen, aiq_result_h* out) {
  if (!c || !q || !gen || !out) return fail(AIQ_ERR_INVALID_ARG, "NULL argument");
  auto t = c->tables.find(table);
  if (t == c->tables.end()) return fail(AIQ_ERR_NOT_FOUND, "unknown table handle");
  auto mi = c->models.find(model);
  if (mi == c->models.end()) return fail(AIQ_ERR_NOT_FOUND, "unknown model handle");
  CUDA_TRY(cudaSetDevice(c->device));
  return run_transform(c, t->second, &mi->second, q, gen, out);
}

aiq_status aiq_run_pair_select(aiq_ctx* c, aiq_table table, int32_t key_column, aiq_model model,
                               const aiq_select* q, aiq_result_h* out) {
  if (!c || !q || !out) return fail(AIQ_ERR_INVALID_ARG, "NULL argument");
  auto t = c->tables.find(table);
  if (t == c->tables.end()) return fail(AIQ_ERR_NOT_FOUND, "unknown table handle");
  if (key_column < 0 || key_column >= static_cast<int32_t>(t->second.cols.size()) ||
      t->second.cols[key_column].type != AIQ_INT64)
    return fail(AIQ_ERR_INVALID_ARG, "key_column must be an INT64 column");
  auto mi = c->models.find(model);
  if (mi == c->models.end()) return fail(AIQ_ERR_NOT_FOUND, "unknown model handle");
  CUDA_TRY(cudaSetDevice(c->device));
  return run_pair_select(c, t->second, key_column, &mi->second, q, out);
}

aiq_status aiq_result(aiq_ctx* c, aiq_result_h h, aiq_result_view* out) {
  if (!c || !out) return fail(AIQ_ERR_INVALID_ARG, "NULL argument");
  auto it = c->results.find(h);
  if (it == c->results.end()) return fail(AIQ_ERR_NOT_FOUND, "unknown result handle");
  *out = it->second.v;
  return AIQ_OK;
}

aiq_status aiq_result_free(aiq_ctx* c, aiq_result_h h) {
  if (!c) return fail(AIQ_ERR_INVALID_ARG, "ctx is NULL");
  auto it = c->results.find(h);
  if (it == c->results.end()) return fail(AIQ_ERR_NOT_FOUND, "unknown result handle");
  c->results.erase(it);
  return AIQ_OK;
}

const char* aiq_last_error(void) { return g_err.c_str(); }

aiq_status aiq_set_option(aiq_ctx* c, const char* name, int64_t value) {
  if (!c || !name) return fail(AIQ_ERR_INVALID_ARG, "NULL argument");
  if (!std::strcmp(name, "token_budget")) {
    if (value < 64 || value > (int64_t(1) << 30)) return fail(AIQ_ERR_INVALID_ARG, "token_budget must be 64..2^30");
    c->token_budget = value;
    return AIQ_OK;
  }
  if (!std::strcmp(name, "profile")) {
    c->profile = value != 0;
    return AIQ_OK;
  }
  if (!std::strcmp(name, "gemm_pair")) {
    c->gemm_pair = value != 0;
    return AIQ_OK;
  }
  if (!std::strcmp(name, "decode_rows")) {
    if (value < 1 || value > (int64_t(1) << 20)) return fail(AIQ_ERR_INVALID_ARG, "decode_rows must be 1..2^20");
    c->decode_rows = value;
    return AIQ_OK;
  }
  if (!std::strcmp(name, "attention_tc")) {
    c->attention_tc = value != 0;
    return AIQ_OK;
  }
  if (!std::strcmp(name, "mlp_split")) {
    c->mlp_split = value < 0 ? -1 : (value != 0);
    return AIQ_OK;
  }
  if (!std::strcmp(name, "device_bytes_max")) {
    // 0 lifts the cap; a cap below what is already allocated only stops growth
    c->bytes_max = value <= 0 ? SIZE_MAX : static_cast<size_t>(value);
    return AIQ_OK;
  }
  return fail(AIQ_ERR_INVALID_ARG, std::string("unknown option ") + name);
}

void* aiq_stream(aiq_ctx* c) { return c ? static_cast<void*>(c->stream) : nullptr; }

aiq_status aiq_kernel_stats(aiq_ctx* c, aiq_kernel_stat* out, int32_t max, int32_t* n_out) {
  if (!c || !n_out || (max > 0 && !out)) return fail(AIQ_ERR_INVALID_ARG, "NULL argument");
  collect_profile(c);
  c->stat_names.clear();
  for (auto& kv : c->stats) c->stat_names.push_back(kv.first);
  int32_t n = 0;
  for (size_t i = 0; i < c->stat_names.size() && n < max; ++i) {
    const StatAcc& s = c->stats[c->stat_names[i]];
    out[n++] = aiq_kernel_stat{c->stat_names[i].c_str(), s.launches, s.ms, s.flops, s.bytes};
  }
  *n_out = n;
  return AIQ_OK;
}

aiq_status aiq_reset_kernel_stats(aiq_ctx* c) {
  if (!c) return fail(AIQ_ERR_INVALID_ARG, "ctx is NULL");
  collect_profile(c);
  c->stats.clear();
  return AIQ_OK;
}

// ------------------------------------------------------------ step ops ---

aiq_status aiq_op_gemm(aiq_ctx* c, const void* A, int64_t lda, const void* B, int64_t ldb, int32_t M, int32_t N,
                       int32_t K, int32_t bn, int32_t epilogue, void* out, int64_t ldo, const int32_t* positions,
                       const float* rope_cos, const float* rope_sin, int32_t rope_cols, int32_t head_dim) {
  if (!c || !A || !B || !out) return fail(AIQ_ERR_INVALID_ARG, "NULL argument");
  if ((epilogue < AIQ_EPI_F16 || epilogue > AIQ_EPI_SWIGLU_F16) && epilogue != AIQ_EPI_RESID_ADD_F32)
    return fail(AIQ_ERR_INVALID_ARG, "unknown epilogue");
  if (M < 0 || N <= 0 || K <= 0 || K % 64 || !(bn == 128 || bn == 256) || N % bn)
    return fail(AIQ_ERR_INVALID_ARG, "need M >= 0, K % 64 == 0, bn in {128, 256}, N % bn == 0");
  if (lda < K || ldb < K) return fail(AIQ_ERR_INVALID_ARG, "lda/ldb smaller than K");
  CUDA_TRY(cudaSetDevice(c->device));
  GemmEpilogue ep;
  ep.kind = epilogue;
  ep.out = out;
  ep.ldo = ldo;
  ep.positions = positions;
  ep.rope_cos = rope_cos;
  ep.rope_sin = rope_sin;
  ep.rope_cols = rope_cols;
  ep.head_dim = head_dim;
  ep.err = c->d_err;
  AIQ_TRY(gemm(c, "op_gemm", static_cast<const __half*>(A), lda, static_cast<const __half*>(B), ldb, M, N, K, bn, ep));
  aiq_status s = sync_and_check(c);
  collect_profile(c);
  return s;
}

aiq_status aiq_op_rope_table(aiq_ctx* c, float* cs, float* sn, int32_t max_pos, int32_t head_dim, float theta) {
  if (!c || !cs || !sn || max_pos <= 0 || head_dim <= 0 || head_dim % 2) return fail(AIQ_ERR_INVALID_ARG, "bad args");
  CUDA_TRY(cudaSetDevice(c->device));
  launch_rope_table(cs, sn, max_pos, head_dim, theta, c->stream);
  return sync_and_check(c);
}

aiq_status aiq_op_rmsnorm(aiq_ctx* c, const float* x, int64_t T, int32_t d, const uint16_t* g, float eps, void* out) {
  if (!c || !x || !g || !out || T < 0 || d <= 0 || d % 4) return fail(AIQ_ERR_INVALID_ARG, "bad args");
  CUDA_TRY(cudaSetDevice(c->device));
  launch_rmsnorm(x, T, d, g, eps, static_cast<__half*>(out), c->d_err, c->stream);
  return sync_and_check(c);
}

aiq_status aiq_op_attention(aiq_ctx* c, const void* qkv, int64_t T, const int32_t* seq_start, int32_t n_seqs,
                            int32_t Hq, int32_t Hkv, int32_t hd, const void* prefix_kv, int32_t P, void* out) {
  if (!c || !qkv || !seq_start || !out || T < 0 || n_seqs < 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv)
    return fail(AIQ_ERR_INVALID_ARG, "bad args");
  if (!(hd == 32 || hd == 64 || hd == 128)) return fail(AIQ_ERR_UNSUPPORTED, "hd must be 32, 64 or 128");
  if (n_seqs == 0 || T == 0) return AIQ_OK;
  CUDA_TRY(cudaSetDevice(c->device));
  int32_t *tile_seq, *tile_q0, *n_tiles;
  const int64_t cap = T / 8 + n_seqs + 1;
  AIQ_TRY(ws(c, "op.tile_seq", cap, &tile_seq));
  AIQ_TRY(ws(c, "op.tile_q0", cap, &tile_q0));
  AIQ_TRY(ws(c, "op.n_tiles", 1, &n_tiles));
  if (P < 0 || (P > 0 && !prefix_kv)) return fail(AIQ_ERR_INVALID_ARG, "bad prefix");
  AIQ_TRY(attention(c, static_cast<const __half*>(qkv), T, n_seqs, seq_start, tile_seq, tile_q0, n_tiles, Hq, Hkv, hd,
                    static_cast<const __half*>(prefix_kv), P, static_cast<__half*>(out)));
  const aiq_status st = sync_and_check(c);
  collect_profile(c);
  return st;
}

aiq_status aiq_op_decode_attention(aiq_ctx* c, const void* qkv, int32_t R, int32_t Hq, int32_t Hkv, int32_t hd,
                                   const void* prefix_kv, int32_t P, const void* own_kv, const int32_t* seq_start,
                                   void* gen_kv, int32_t gen_cap, int32_t slot, void* out) {
  if (!c || !qkv || !own_kv || !seq_start || !gen_kv || !out || R < 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv ||
      P < 0 || (P > 0 && !prefix_kv) || gen_cap < 1 || slot < 0 || slot >= gen_cap)
    return fail(AIQ_ERR_INVALID_ARG, "bad args");
  if (!(hd == 32 || hd == 64 || hd == 128) || Hq / Hkv > 8)
    return fail(AIQ_ERR_UNSUPPORTED, "hd must be 32, 64 or 128 and Hq / Hkv <= 8");
  if (R == 0) return AIQ_OK;
  CUDA_TRY(cudaSetDevice(c->device));
  const int e = launch_decode_attention(static_cast<const __half*>(qkv), static_cast<int64_t>(Hq + 2 * Hkv) * hd, R,
                                        Hq, Hkv, hd, static_cast<const __half*>(prefix_kv), P,
                                        static_cast<const __half*>(own_kv), seq_start, static_cast<__half*>(gen_kv),
                                        gen_cap, slot, static_cast<__half*>(out), c->d_err, c->stream);
  if (e != 0) return fail(AIQ_ERR_CUDA, std::string("decode attention launch: ") +
                                            cudaGetErrorString(static_cast<cudaError_t>(e)));
  return sync_and_check(c);
}

aiq_status aiq_op_wait_expiry_selftest(aiq_ctx* c, uint64_t limit_ns) {
  if (!c || limit_ns < 1000 || limit_ns > 1000000000ull) return fail(AIQ_ERR_INVALID_ARG, "bad args");
  CUDA_TRY(cudaSetDevice(c->device));
  const int e = launch_wait_expiry(limit_ns, c->d_err, c->stream);
  if (e != 0) return fail(AIQ_ERR_CUDA, std::string("wait self-test launch: ") +
                                            cudaGetErrorString(static_cast<cudaError_t>(e)));
  return sync_and_check(c);
}

}  // extern "C"
