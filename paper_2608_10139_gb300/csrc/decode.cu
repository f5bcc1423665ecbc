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
// of the row's keys.  Warp w takes key blocks w, w + 8, ... of KB keys.  In a
// block every lane (a pair of lanes for head_dim 128) holds one key: the key
// row and all KB value rows of the block are loaded together, so a block costs
// one memory round trip; the scores of the G heads come from q in shared
// memory, then P V accumulates with each lane owning HD / 32 output columns.
// The eight warps' partial (max, sum, output) are merged at the end.
template <int HD, int G>
__global__ void __launch_bounds__(kDecThreads) k_decode_attention(DecArgs a) {
  constexpr int NW = kDecThreads / 32;
  constexpr int DPL = HD / 32;           // output columns per lane
  constexpr int LPK = HD == 128 ? 2 : 1; // lanes per key
  constexpr int KB = 32 / LPK;           // keys per warp block
  constexpr int KC = HD / 8 / LPK;       // 16-byte chunks of a key row per lane
  constexpr int VW = (DPL + 1) / 2;      // 32-bit words of packed halves per value slice
  __shared__ __align__(16) float sq[G * HD];
  __shared__ float sp[NW][G][KB];
  __shared__ float sm_m[NW][G], sm_l[NW][G];
  __shared__ __align__(16) float so[NW][G * HD];

  const int r = blockIdx.x / a.Hkv, h = blockIdx.x % a.Hkv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
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
  float m_run[G], l_lane[G], o[G][DPL];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m_run[g] = -INFINITY;
    l_lane[g] = 0.f;
#pragma unroll
    for (int e = 0; e < DPL; ++e) o[g][e] = 0.f;
  }
  const int kslot = lane / LPK, part = lane % LPK;  // this lane's key in the block, its half of the row

  for (int blk = warp; blk * KB < n_keys; blk += NW) {
    const int j = blk * KB + kslot;
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
    const int nvalid = min(KB, n_keys - blk * KB);
    // issue every load of the block: this lane's part of its key row, and its
    // column slice of all KB value rows (plain loads: the newest slot was
    // written by this block a moment ago)
    uint4 kr[KC];
    if (valid) {
#pragma unroll
      for (int c = 0; c < KC; ++c) kr[c] = reinterpret_cast<const uint4*>(krow + part * (HD / 2))[c];
    } else {
#pragma unroll
      for (int c = 0; c < KC; ++c) kr[c] = make_uint4(0u, 0u, 0u, 0u);
    }
    const unsigned long long my_v = reinterpret_cast<unsigned long long>(krow ? krow + kd : nullptr);
    uint32_t vr[KB][VW];
#pragma unroll
    for (int jb = 0; jb < KB; ++jb) {
      const __half* vrow = reinterpret_cast<const __half*>(__shfl_sync(0xffffffffu, my_v, jb * LPK));
      if (jb < nvalid) {
        if constexpr (DPL == 1) {
          vr[jb][0] = reinterpret_cast<const uint16_t*>(vrow)[lane];
        } else if constexpr (DPL == 2) {
          vr[jb][0] = reinterpret_cast<const uint32_t*>(vrow)[lane];
        } else {
          const uint2 u = reinterpret_cast<const uint2*>(vrow)[lane];
          vr[jb][0] = u.x;
          vr[jb][1] = u.y;
        }
      } else {
#pragma unroll
        for (int e = 0; e < VW; ++e) vr[jb][e] = 0u;
      }
    }
    // scores of the G heads for this lane's key (partial over its half of the row for hd 128)
    float s[G];
#pragma unroll
    for (int g = 0; g < G; ++g) s[g] = 0.f;
#pragma unroll
    for (int c = 0; c < KC; ++c) {
      const __half2* k2 = reinterpret_cast<const __half2*>(&kr[c]);
      float kf[8];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = __half22float2(k2[e]);
        kf[2 * e] = f.x;
        kf[2 * e + 1] = f.y;
      }
      const int d0 = part * (HD / 2) + 8 * c;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float4 q0 = *reinterpret_cast<const float4*>(&sq[g * HD + d0]);
        const float4 q1 = *reinterpret_cast<const float4*>(&sq[g * HD + d0 + 4]);
        s[g] += q0.x * kf[0] + q0.y * kf[1] + q0.z * kf[2] + q0.w * kf[3] + q1.x * kf[4] + q1.y * kf[5] +
                q1.z * kf[6] + q1.w * kf[7];
      }
    }
#pragma unroll
    for (int g = 0; g < G; ++g) {
      if constexpr (LPK == 2) s[g] += __shfl_xor_sync(0xffffffffu, s[g], 1);
      const float sv = valid ? s[g] : -INFINITY;
      const float m_new = fmaxf(m_run[g], warp_max(sv));  // finite: the block's first key is valid
      const float f = exp2f(m_run[g] - m_new);
      const float p = valid ? exp2f(sv - m_new) : 0.f;
      l_lane[g] = l_lane[g] * f + (part == 0 ? p : 0.f);
#pragma unroll
      for (int e = 0; e < DPL; ++e) o[g][e] *= f;
      m_run[g] = m_new;
      if (part == 0) sp[warp][g][kslot] = p;
    }
    __syncwarp();
#pragma unroll
    for (int jb = 0; jb < KB; ++jb) {
      float vf[DPL];
      if constexpr (DPL == 1) {
        vf[0] = __half2float(__ushort_as_half(static_cast<unsigned short>(vr[jb][0])));
      } else {
#pragma unroll
        for (int e = 0; e < VW; ++e) {
          const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&vr[jb][e]));
          vf[2 * e] = f.x;
          vf[2 * e + 1] = f.y;
        }
      }
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float p = sp[warp][g][jb];  // 0 for keys past the end
#pragma unroll
        for (int e = 0; e < DPL; ++e) o[g][e] += p * vf[e];
      }
    }
    __syncwarp();
  }

  // merge the warps' partial softmax states
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const float l = warp_sum(l_lane[g]);
    if (lane == 0) {
      sm_m[warp][g] = m_run[g];
      sm_l[warp][g] = l;
    }
#pragma unroll
    for (int e = 0; e < DPL; ++e) so[warp][g * HD + lane * DPL + e] = o[g][e];
  }
  __syncthreads();
  __half* orow = a.out + static_cast<int64_t>(r) * a.Hq * HD + h * G * HD;
  for (int i = tid; i < G * HD; i += kDecThreads) {
    const int g = i / HD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < NW; ++w) M = fmaxf(M, sm_m[w][g]);
    float L = 0.f, O = 0.f;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
      const float f = sm_m[w][g] == -INFINITY ? 0.f : exp2f(sm_m[w][g] - M);  // a warp without keys
      L += sm_l[w][g] * f;
      O += so[w][i] * f;
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

template <int HD, int G>
int launch_dec(const DecArgs& a, int R, cudaStream_t s) {
  k_decode_attention<HD, G><<<R * a.Hkv, kDecThreads, 0, s>>>(a);
  return cudaGetLastError();
}

template <int HD>
int launch_dec_g(const DecArgs& a, int R, cudaStream_t s) {
  switch (a.G) {
    case 1: return launch_dec<HD, 1>(a, R, s);
    case 2: return launch_dec<HD, 2>(a, R, s);
    case 4: return launch_dec<HD, 4>(a, R, s);
    case 8: return launch_dec<HD, 8>(a, R, s);
  }
  return cudaErrorInvalidValue;
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
    case 32: return launch_dec_g<32>(a, R, s);
    case 64: return launch_dec_g<64>(a, R, s);
    default: return launch_dec_g<128>(a, R, s);
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
