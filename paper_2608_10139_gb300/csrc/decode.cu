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

constexpr int kDecThreads = 128;  // 4 warps per (row, KV head)
constexpr int kDecMaxG = 8;       // query heads per KV head

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

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One block per (row, KV head): the G query heads of the group against all
// of the row's keys.  Warp w takes key blocks w, w + 4, ... of 32 keys; in a
// block each lane scores one key for all G heads (q from shared memory),
// then the warp accumulates P V with each lane owning HD / 32 output columns.
// The four warps' partial (max, sum, output) are merged at the end.
template <int HD>
__global__ void __launch_bounds__(kDecThreads) k_decode_attention(DecArgs a) {
  constexpr int DPL = HD / 32;  // output columns per lane
  __shared__ __align__(16) float sq[kDecMaxG * HD];
  __shared__ float sp[4][kDecMaxG][32];
  __shared__ float sm_m[4][kDecMaxG], sm_l[4][kDecMaxG];
  __shared__ __align__(16) float so[4][kDecMaxG][HD];

  const int r = blockIdx.x / a.Hkv, h = blockIdx.x % a.Hkv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = a.G;
  const int kd = a.Hkv * HD;
  const int64_t ld = 2 * static_cast<int64_t>(kd);
  const __half* qrow = a.qkv + static_cast<int64_t>(r) * a.ldq;
  const int st = a.seq_start[r], len = a.seq_start[r + 1] - st;
  __half* slot = a.gkv + (static_cast<int64_t>(r) * a.gcap + a.slot) * ld;

  // this token's key and value into its cache slot; its G query heads (scaled) into shared memory
  for (int i = tid; i < HD / 8; i += kDecThreads) {
    reinterpret_cast<uint4*>(slot + h * HD)[i] = reinterpret_cast<const uint4*>(qrow + (a.Hq + h) * HD)[i];
    reinterpret_cast<uint4*>(slot + kd + h * HD)[i] =
        reinterpret_cast<const uint4*>(qrow + (a.Hq + a.Hkv + h) * HD)[i];
  }
  for (int i = tid; i < G * HD; i += kDecThreads) sq[i] = __half2float(qrow[h * G * HD + i]) * a.scale_log2;
  __syncthreads();  // the slot written above is read back by this block below

  const int n_keys = a.P + len + a.slot + 1;
  float m_run[kDecMaxG], l_lane[kDecMaxG], o[kDecMaxG][DPL];
#pragma unroll
  for (int g = 0; g < kDecMaxG; ++g) {
    m_run[g] = -INFINITY;
    l_lane[g] = 0.f;
#pragma unroll
    for (int e = 0; e < DPL; ++e) o[g][e] = 0.f;
  }

  for (int blk = warp; blk * 32 < n_keys; blk += 4) {
    const int j = blk * 32 + lane;
    const bool valid = j < n_keys;
    // key row of key j: shared prefix, then the row's prompt, then its generated tokens
    const __half* krow = nullptr;
    if (valid) {
      if (j < a.P)
        krow = a.pkv + j * ld;
      else if (j < a.P + len)
        krow = a.kvc + (st + j - a.P) * ld;
      else
        krow = a.gkv + (static_cast<int64_t>(r) * a.gcap + (j - a.P - len)) * ld;
      krow += h * HD;
    }
    float s[kDecMaxG];
#pragma unroll
    for (int g = 0; g < kDecMaxG; ++g) s[g] = 0.f;
    if (valid) {
#pragma unroll
      for (int c = 0; c < HD / 8; ++c) {
        // plain loads: this block wrote the newest slot a moment ago
        const uint4 kv = reinterpret_cast<const uint4*>(krow)[c];
        const __half2* k2 = reinterpret_cast<const __half2*>(&kv);
        float kf[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __half22float2(k2[e]);
          kf[2 * e] = f.x;
          kf[2 * e + 1] = f.y;
        }
#pragma unroll
        for (int g = 0; g < kDecMaxG; ++g) {
          if (g < G) {
            const float4 q0 = *reinterpret_cast<const float4*>(&sq[g * HD + 8 * c]);
            const float4 q1 = *reinterpret_cast<const float4*>(&sq[g * HD + 8 * c + 4]);
            s[g] += q0.x * kf[0] + q0.y * kf[1] + q0.z * kf[2] + q0.w * kf[3] + q1.x * kf[4] + q1.y * kf[5] +
                    q1.z * kf[6] + q1.w * kf[7];
          }
        }
      }
    }
#pragma unroll
    for (int g = 0; g < kDecMaxG; ++g) {
      if (g < G) {
        const float sv = valid ? s[g] : -INFINITY;
        const float m_new = fmaxf(m_run[g], warp_max(sv));  // finite: key blk * 32 is valid
        const float f = exp2f(m_run[g] - m_new);
        const float p = valid ? exp2f(sv - m_new) : 0.f;
        l_lane[g] = l_lane[g] * f + p;
#pragma unroll
        for (int e = 0; e < DPL; ++e) o[g][e] *= f;
        m_run[g] = m_new;
        sp[warp][g][lane] = p;
      }
    }
    __syncwarp();
    const int nvalid = min(32, n_keys - blk * 32);
    const unsigned long long my_v = reinterpret_cast<unsigned long long>(krow ? krow + kd : nullptr);
#pragma unroll 4
    for (int jj = 0; jj < nvalid; ++jj) {
      const __half* vrow = reinterpret_cast<const __half*>(__shfl_sync(0xffffffffu, my_v, jj));
      float vf[DPL];
      if constexpr (DPL == 1) {
        vf[0] = __half2float(vrow[lane]);
      } else if constexpr (DPL == 2) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2*>(vrow + 2 * lane));
        vf[0] = f.x;
        vf[1] = f.y;
      } else {
        const uint2 u = *reinterpret_cast<const uint2*>(vrow + 4 * lane);
        const float2 f0 = __half22float2(*reinterpret_cast<const __half2*>(&u.x));
        const float2 f1 = __half22float2(*reinterpret_cast<const __half2*>(&u.y));
        vf[0] = f0.x;
        vf[1] = f0.y;
        vf[2] = f1.x;
        vf[3] = f1.y;
      }
#pragma unroll
      for (int g = 0; g < kDecMaxG; ++g) {
        if (g < G) {
          const float p = sp[warp][g][jj];
#pragma unroll
          for (int e = 0; e < DPL; ++e) o[g][e] += p * vf[e];
        }
      }
    }
    __syncwarp();
  }

  // merge the four warps' partial softmax states
#pragma unroll
  for (int g = 0; g < kDecMaxG; ++g) {
    if (g < G) {
      const float l = warp_sum(l_lane[g]);
      if (lane == 0) {
        sm_m[warp][g] = m_run[g];
        sm_l[warp][g] = l;
      }
#pragma unroll
      for (int e = 0; e < DPL; ++e) so[warp][g][lane * DPL + e] = o[g][e];
    }
  }
  __syncthreads();
  __half* orow = a.out + static_cast<int64_t>(r) * a.Hq * HD + h * G * HD;
  for (int i = tid; i < G * HD; i += kDecThreads) {
    const int g = i / HD, dd = i % HD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, sm_m[w][g]);
    float L = 0.f, O = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float f = sm_m[w][g] == -INFINITY ? 0.f : exp2f(sm_m[w][g] - M);  // a warp without keys
      L += sm_l[w][g] * f;
      O += so[w][g][dd] * f;
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
  k_decode_attention<HD><<<R * a.Hkv, kDecThreads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace

int launch_decode_attention(const __half* qkv, int64_t ldq, int R, int Hq, int Hkv, int hd, const __half* pkv, int P,
                            const __half* kvc, const int32_t* seq_start, __half* gkv, int gcap, int slot, __half* out,
                            int* err, cudaStream_t s) {
  if (R <= 0) return 0;
  if (Hq % Hkv || Hq / Hkv > kDecMaxG || !(hd == 32 || hd == 64 || hd == 128) || slot < 0 || slot >= gcap)
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
