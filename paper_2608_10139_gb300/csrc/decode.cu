// Generation (AI_TRANSFORM, Table 1: causal-LM forward with generative
// decoding, output masked with a pad id) and the on-device LIKE match of
// Table 2 Q5.
//
// After a chunk's prefill, every row of the chunk decodes together: one new
// token per row per step.  A step is the decoder over R single-token rows
// (the prefill GEMMs with M = R), this file's decode attention over each
// row's cached keys (shared prefix, the row's own prompt tokens, the tokens it
// generated so far), the final RMSNorm and the full-vocabulary LM head, whose
// GEMM epilogue keeps only each row's (max logit, first index) through a
// 64-bit atomicMax; k_decode_select turns that into the next token.
#include "common.cuh"
#include "kernels.h"

namespace aiq {
namespace {

constexpr int kDecThreads = 256;  // 8 warps per (row, KV head)

struct DecArgs {
  const __half* qkv;  // [R][ldq]: q heads, k heads, v heads of this step's token
  int64_t ldq;
  int Hq, Hkv, G;
  const __half* pkv;  // [P][2 kd] shared-prefix keys | values (may be null when P == 0)
  int P;
  const __half* kvc;  // [Tc][2 kd] the rows' own prompt keys | values
  const int32_t* seq_start;  // [R + 1] row r's prompt tokens are kvc rows seq_start[r] ..
  __half* gkv;        // [R][gcap][2 kd] generated tokens' keys | values
  int gcap;
  int slot;           // this step's token goes to gkv slot `slot`; it attends slots 0..slot
  float scale_log2;   // log2(e) / sqrt(hd)
  __half* out;        // [R][Hq hd]
  int* err;
};

__device__ __forceinline__ void cp_async16(uint32_t saddr, const void* gmem, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(saddr), "l"(gmem), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t saddr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(saddr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], uint32_t saddr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(saddr));
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&x)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(x[0]), "r"(x[1]), "r"(x[2]), "r"(x[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_h2(float x, float y) {
  __half2 v = __floats2half2_rn(x, y);
  return *reinterpret_cast<uint32_t*>(&v);
}

template <int HD>
struct DecCfg {
  static constexpr int NW = kDecThreads / 32;
  static constexpr int KB = HD == 128 ? 16 : 32;  // keys per warp block
  static constexpr int LDS = HD + 8;    // padded smem row (halves): conflict-free ldmatrix
  static constexpr int WARP_HALVES = 2 * KB * LDS;  // K block then V block
  static constexpr int SMEM = NW * WARP_HALVES * 2;
};

// One block per (row, KV head): the G <= 8 query heads of the group against
// all of the row's keys, on m16n8k16 tensor-core MMAs (the heads are the
// rows of the A tile, the rest of its 16 rows are zero).  Warp w takes key
// blocks w, w + 8, ... of 32 keys (16 at head_dim 128): it stages a block's K
// and V rows in its own shared-memory slice with cp.async (all rows of both at
// once), then
// S = Q K^T, the online softmax on the accumulator fragments and O += P V
// with V read through ldmatrix.trans.  The eight warps' partial (max, sum,
// output) are merged at the end.
template <int HD>
__global__ void __launch_bounds__(kDecThreads, HD == 128 ? 2 : 3) k_decode_attention(DecArgs a) {
  using C = DecCfg<HD>;
  constexpr int NW = C::NW, KB = C::KB, LDS = C::LDS;
  constexpr int KS = HD / 16;  // k-steps of Q K^T
  constexpr int DN = HD / 8;   // 8-wide output column tiles
  constexpr int CH = HD / 8;   // 16-byte chunks per row
  extern __shared__ __align__(16) uint8_t smem_raw[];

  const int r = blockIdx.x / a.Hkv, h = blockIdx.x % a.Hkv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = a.G;
  const int kd = a.Hkv * HD;
  const int64_t ld = 2 * static_cast<int64_t>(kd);
  const __half* qrow = a.qkv + static_cast<int64_t>(r) * a.ldq;
  const int st = a.seq_start[r], len = a.seq_start[r + 1] - st;
  __half* slot = a.gkv + (static_cast<int64_t>(r) * a.gcap + a.slot) * ld;
  __half* sK = reinterpret_cast<__half*>(smem_raw) + warp * C::WARP_HALVES;
  __half* sV = sK + KB * LDS;

  // this token's key and value into its cache slot, for the later steps; this
  // step reads them straight from the qkv row (no wait on the store)
  for (int i = tid; i < HD / 8; i += kDecThreads) {
    reinterpret_cast<uint4*>(slot + h * HD)[i] = reinterpret_cast<const uint4*>(qrow + (a.Hq + h) * HD)[i];
    reinterpret_cast<uint4*>(slot + kd + h * HD)[i] =
        reinterpret_cast<const uint4*>(qrow + (a.Hq + a.Hkv + h) * HD)[i];
  }

  const int n_keys = a.P + len + a.slot + 1;
  const int gq = lane >> 2, tq = lane & 3;
  // A fragments of the query tile straight from global memory: row gq is query
  // head h G + gq (rows >= G and 8..15 are zero padding)
  uint32_t qf[KS][4];
  {
    const uint32_t* q32 = reinterpret_cast<const uint32_t*>(qrow + (h * G + gq) * HD);
#pragma unroll
    for (int kk = 0; kk < KS; ++kk) {
      qf[kk][0] = gq < G ? q32[(kk * 16 + 2 * tq) / 2] : 0u;
      qf[kk][1] = 0u;
      qf[kk][2] = gq < G ? q32[(kk * 16 + 8 + 2 * tq) / 2] : 0u;
      qf[kk][3] = 0u;
    }
  }
  float o[DN][4];
#pragma unroll
  for (int i = 0; i < DN; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m0 = -INFINITY, l0 = 0.f;  // row gq (a head when gq < G); rows 8..15 are padding

  for (int blk = warp; blk * KB < n_keys; blk += NW) {
    const int key0 = blk * KB;
    // stage K and V of keys key0 .. key0 + KB - 1: shared prefix, the row's prompt, its generated tokens
#pragma unroll
    for (int i = 0; i < KB * CH / 32; ++i) {
      const int c = lane + 32 * i;
      const int kr = c / CH, part = c % CH;
      const int j = key0 + kr;
      const bool valid = j < n_keys;
      const __half* krow;
      if (valid) {
        if (j < a.P)
          krow = a.pkv + j * ld;
        else if (j < a.P + len)
          krow = a.kvc + (st + j - a.P) * ld;
        else if (j < n_keys - 1)
          krow = a.gkv + (static_cast<int64_t>(r) * a.gcap + (j - a.P - len)) * ld;
        else
          krow = qrow + a.Hq * HD;  // this step's token: its k heads, then (kd further) its v heads
        krow += h * HD;
      } else {
        krow = qrow;  // zero-filled chunk: any mapped address
      }
      cp_async16(smem_u32(sK + kr * LDS + part * 8), krow + part * 8, valid);
      cp_async16(smem_u32(sV + kr * LDS + part * 8), krow + kd + part * 8, valid);
    }
    cp_async_wait_all();
    __syncwarp();
    float sc[KB / 8][4];
#pragma unroll
    for (int n = 0; n < KB / 8; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < KS; ++kk) {
#pragma unroll
      for (int np = 0; np < KB / 16; ++np) {
        const int mat = lane >> 3;
        const int key = np * 16 + (lane & 7) + 8 * (mat >> 1);
        const int dim = kk * 16 + 8 * (mat & 1);
        uint32_t bb[4];
        ldsm_x4(bb, smem_u32(sK + key * LDS + dim));
        mma16816(sc[2 * np], qf[kk], bb[0], bb[1]);
        mma16816(sc[2 * np + 1], qf[kk], bb[2], bb[3]);
      }
    }
    // log2 units, keys past the end masked; row gq uses elements 0 and 1
    float mx = -INFINITY;
#pragma unroll
    for (int n = 0; n < KB / 8; ++n) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int key = key0 + n * 8 + 2 * tq + e;
        const float v = key < n_keys ? sc[n][e] * a.scale_log2 : -INFINITY;
        sc[n][e] = v;
        mx = fmaxf(mx, v);
      }
    }
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
    const float mn = fmaxf(m0, mx);  // finite: key0 < n_keys
    const float c0 = exp2f(m0 - mn);
    m0 = mn;
    float rs = 0.f;
#pragma unroll
    for (int n = 0; n < KB / 8; ++n) {
      sc[n][0] = exp2f(sc[n][0] - mn);
      sc[n][1] = exp2f(sc[n][1] - mn);
      rs += sc[n][0] + sc[n][1];
    }
    l0 = l0 * c0 + rs;
#pragma unroll
    for (int i = 0; i < DN; ++i) {
      o[i][0] *= c0;
      o[i][1] *= c0;
    }
#pragma unroll
    for (int k2 = 0; k2 < KB / 16; ++k2) {
      uint32_t pa[4];
      pa[0] = pack_h2(sc[2 * k2][0], sc[2 * k2][1]);
      pa[1] = 0u;  // padding rows 8..15
      pa[2] = pack_h2(sc[2 * k2 + 1][0], sc[2 * k2 + 1][1]);
      pa[3] = 0u;
#pragma unroll
      for (int dp = 0; dp < DN / 2; ++dp) {
        const int mat = lane >> 3;
        const int key = k2 * 16 + (lane & 7) + 8 * (mat & 1);
        const int dim = dp * 16 + 8 * (mat >> 1);
        uint32_t bb[4];
        ldsm_x4_t(bb, smem_u32(sV + key * LDS + dim));
        mma16816(o[2 * dp], pa, bb[0], bb[1]);
        mma16816(o[2 * dp + 1], pa, bb[2], bb[3]);
      }
    }
    __syncwarp();  // every lane is done with this warp's staging before it is refilled
  }
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);

  // merge the warps' partial softmax states (the staging area is reused)
  __syncthreads();
  float* mm = reinterpret_cast<float*>(smem_raw);  // [NW][8] max, [NW][8] sum, [NW][8][HD]
  float* ll = mm + NW * 8;
  float* oo = ll + NW * 8;
  if (tq == 0) {
    mm[warp * 8 + gq] = m0;
    ll[warp * 8 + gq] = l0;
  }
#pragma unroll
  for (int i = 0; i < DN; ++i) {
    oo[(warp * 8 + gq) * HD + i * 8 + 2 * tq] = o[i][0];
    oo[(warp * 8 + gq) * HD + i * 8 + 2 * tq + 1] = o[i][1];
  }
  __syncthreads();
  __half* orow = a.out + static_cast<int64_t>(r) * a.Hq * HD + h * G * HD;
  for (int i = tid; i < G * HD; i += kDecThreads) {
    const int g = i / HD, dd = i % HD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < NW; ++w) M = fmaxf(M, mm[w * 8 + g]);
    float L = 0.f, O = 0.f;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const float f = mm[w * 8 + g] == -INFINITY ? 0.f : exp2f(mm[w * 8 + g] - M);  // a warp without keys
      L += ll[w * 8 + g] * f;
      O += oo[(w * 8 + g) * HD + dd] * f;
    }
    orow[i] = __float2half_rn(O / L);
  }
}

// Next token of each row from the LM head's packed (max, first index), the
// pad mask after an eos, and the position the token takes when fed back.
__global__ void k_decode_select(unsigned long long* best, int R, int t, int max_new, int eos, int pad, int V,
                                int32_t* done, int32_t* gen_tok, int32_t* gen_len, int32_t* next_tok, int32_t* pos,
                                const int32_t* seq_start, int P, int* err) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= R) return;
  const unsigned long long key = best[r];
  best[r] = 0ull;  // ready for the next step's atomicMax
  int tok = static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFull));
  if (key == 0ull || tok < 0 || tok >= V) {
    set_dev_error(err, DEVERR_BOUNDS);
    tok = 0;
  }
  const int was_done = t == 0 ? 0 : done[r];
  if (t == 0) gen_len[r] = max_new;
  gen_tok[static_cast<int64_t>(r) * max_new + t] = was_done ? pad : tok;
  if (!was_done && tok == eos) gen_len[r] = t;
  done[r] = was_done || tok == eos;
  next_tok[r] = tok;
  pos[r] = P + (seq_start[r + 1] - seq_start[r]) + t;
}

// Rows of a chunk whose text is empty take the shared prefix's last hidden state.
__global__ void k_patch_empty_rows(float* resid, const int32_t* last_idx, const float* prefix_last, int R, int d) {
  const int r = blockIdx.x;
  if (r >= R || last_idx[r] >= 0) return;
  for (int i = threadIdx.x; i < d; i += blockDim.x) resid[static_cast<int64_t>(r) * d + i] = prefix_last[i];
}

// fp32 LM-head bias, -inf on the padding columns [V, Vpad).
__global__ void k_bias_f32(const uint16_t* b, int V, int Vpad, float* out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= Vpad) return;
  out[i] = i < V ? __uint_as_float(static_cast<uint32_t>(b[i]) << 16) : -INFINITY;
}

// Table 2 Q5: does row r's generated text (its tokens before the eos)
// contain the pattern as a contiguous run?  An empty pattern matches.
__global__ void k_like_match(const int32_t* gen_tok, const int32_t* gen_len, int64_t S, int max_new,
                             const int32_t* pattern, int plen, int32_t* match) {
  const int64_t r = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (r >= S) return;
  const int32_t* t = gen_tok + r * max_new;
  const int n = gen_len[r];
  int hit = plen == 0;
  for (int i = 0; !hit && i + plen <= n; ++i) {
    int k = 0;
    while (k < plen && t[i + k] == pattern[k]) ++k;
    hit = k == plen;
  }
  match[r] = hit;
}

// out[k] = rows[pos[k]] of a [*, width] int32 matrix.
__global__ void k_gather_rows_i32(const int32_t* src, int width, const int32_t* pos, int64_t n, int32_t* out) {
  const int64_t k = blockIdx.x;
  if (k >= n) return;
  const int32_t* s = src + static_cast<int64_t>(pos[k]) * width;
  for (int i = threadIdx.x; i < width; i += blockDim.x) out[k * width + i] = s[i];
}

template <int HD>
int launch_dec(const DecArgs& a, int R, cudaStream_t s) {
  using C = DecCfg<HD>;
  cudaError_t e = cudaFuncSetAttribute(k_decode_attention<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  k_decode_attention<HD><<<R * a.Hkv, kDecThreads, C::SMEM, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

int launch_decode_attention(const __half* qkv, int64_t ldq, int R, int Hq, int Hkv, int hd, const __half* pkv, int P,
                            const __half* kvc, const int32_t* seq_start, __half* gkv, int gcap, int slot, __half* out,
                            int* err, cudaStream_t s) {
  if (R <= 0) return 0;
  const int G = Hkv > 0 ? Hq / Hkv : 0;
  if (Hkv <= 0 || Hq % Hkv || !(G == 1 || G == 2 || G == 4 || G == 8) || !(hd == 32 || hd == 64 || hd == 128) ||
      slot < 0 || slot >= gcap)
    return cudaErrorInvalidValue;
  DecArgs a{qkv, ldq, Hq, Hkv, Hq / Hkv, pkv, P, kvc, seq_start, gkv, gcap, slot,
            1.4426950408889634f / sqrtf(static_cast<float>(hd)), out, err};
  switch (hd) {
    case 32: return launch_dec<32>(a, R, s);
    case 64: return launch_dec<64>(a, R, s);
    default: return launch_dec<128>(a, R, s);
  }
}

void launch_decode_select(unsigned long long* best, int R, int t, int max_new, int eos, int pad, int V, int32_t* done,
                          int32_t* gen_tok, int32_t* gen_len, int32_t* next_tok, int32_t* pos,
                          const int32_t* seq_start, int P, int* err, cudaStream_t s) {
  if (R <= 0) return;
  k_decode_select<<<(R + 255) / 256, 256, 0, s>>>(best, R, t, max_new, eos, pad, V, done, gen_tok, gen_len, next_tok,
                                                  pos, seq_start, P, err);
}

void launch_patch_empty_rows(float* resid, const int32_t* last_idx, const float* prefix_last, int R, int d,
                             cudaStream_t s) {
  if (R <= 0) return;
  k_patch_empty_rows<<<R, 128, 0, s>>>(resid, last_idx, prefix_last, R, d);
}

void launch_bias_f32(const uint16_t* b, int V, int Vpad, float* out, cudaStream_t s) {
  k_bias_f32<<<(Vpad + 255) / 256, 256, 0, s>>>(b, V, Vpad, out);
}

void launch_like_match(const int32_t* gen_tok, const int32_t* gen_len, int64_t S, int max_new, const int32_t* pattern,
                       int plen, int32_t* match, cudaStream_t s) {
  if (S <= 0) return;
  k_like_match<<<static_cast<unsigned>((S + 127) / 128), 128, 0, s>>>(gen_tok, gen_len, S, max_new, pattern, plen,
                                                                     match);
}

void launch_gather_rows_i32(const int32_t* src, int width, const int32_t* pos, int64_t n, int32_t* out,
                            cudaStream_t s) {
  if (n <= 0) return;
  k_gather_rows_i32<<<static_cast<unsigned>(n), 128, 0, s>>>(src, width, pos, n, out);
}

}  // namespace aiq
