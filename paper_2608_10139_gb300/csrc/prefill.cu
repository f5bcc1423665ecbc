// Memory-bound steps of the decoder prefill: weight conversion at load,
// rotary-embedding table, token-embedding gather, RMSNorm, and the label head
// that reads only the label rows of the LM head at each row's last token
// (Fig. 2 slices logits[:, -1, :] at the label ids; the full vocabulary row is
// never formed).
#include "common.cuh"
#include "kernels.h"

namespace aiq {
namespace {

__device__ __forceinline__ float bf16_bits_to_float(uint16_t b) {
  return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

// dst row r of a [rows, cols] fp16 matrix from a bf16 source.  With an
// interleave block ib > 0, the source holds two stacked [half_rows, cols]
// matrices (gate then up) and dst rows alternate blocks of ib gate rows and
// ib up rows, so that one GEMM output tile holds matching gate/up columns.
__global__ void k_bf16_to_f16(const uint16_t* src, __half* dst, int64_t rows, int64_t cols, int ib, int64_t half_rows,
                              int64_t ldd, int* err) {
  const int64_t n = rows * cols;
  bool bad = false;
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = e / cols, c = e - r * cols;
    int64_t sr = r;
    if (ib > 0) {
      const int64_t b = r / (2 * ib), w = r % (2 * ib);
      sr = w < ib ? b * ib + w : half_rows + b * ib + (w - ib);
    }
    const float v = bf16_bits_to_float(src[sr * cols + c]);
    bad |= !(fabsf(v) <= 65504.f);
    dst[r * ldd + c] = __float2half_rn(v);
  }
  if (bad) set_dev_error(err, DEVERR_FP16_RANGE);
}

__global__ void k_rope_table(float* cos_t, float* sin_t, int max_pos, int hd, double theta) {
  const int half = hd / 2;
  const int64_t n = static_cast<int64_t>(max_pos) * half;
  for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int p = static_cast<int>(e / half), i = static_cast<int>(e % half);
    const double inv = pow(theta, -2.0 * i / hd);
    const double a = p * inv;
    cos_t[e] = static_cast<float>(cos(a));
    sin_t[e] = static_cast<float>(sin(a));
  }
}

// One warp per token; 8 bf16 (16 bytes) per lane per step.  With xh / ss the
// row is also written as fp16, times the first layer's attention-norm gain
// when `gain` is given (the fused RMSNorm's input), and its sums of squares
// per 128 columns (16 lanes x 8 values, of the unscaled row) are stored, in a
// fixed order.
__global__ void k_embed(const int32_t* tok, int64_t T, const uint16_t* emb, int d, float* resid, __half* xh, float* ss,
                        const uint16_t* gain, int* err) {
  const int64_t t = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (t >= T) return;
  const uint4* src = reinterpret_cast<const uint4*>(emb + static_cast<int64_t>(tok[t]) * d);
  float4* dst = reinterpret_cast<float4*>(resid + t * d);
  bool bad = false;
  for (int c0 = 0; c0 < d / 8; c0 += 32) {
    const int c = c0 + lane;
    float f[8];
    float part = 0.f;
    if (c < d / 8) {
      const uint4 v = src[c];
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        f[2 * j] = __uint_as_float(w[j] << 16);
        f[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
      }
      dst[2 * c] = make_float4(f[0], f[1], f[2], f[3]);
      dst[2 * c + 1] = make_float4(f[4], f[5], f[6], f[7]);
      if (xh) {
        uint32_t pk[4];
        float gf[8] = {1.f, 1.f, 1.f, 1.f, 1.f, 1.f, 1.f, 1.f};
        if (gain) {
          const uint4 gv = reinterpret_cast<const uint4*>(gain)[c];
          const uint32_t gw[4] = {gv.x, gv.y, gv.z, gv.w};
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            gf[2 * j] = __uint_as_float(gw[j] << 16);
            gf[2 * j + 1] = __uint_as_float(gw[j] & 0xFFFF0000u);
          }
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float a = f[2 * j] * gf[2 * j], b = f[2 * j + 1] * gf[2 * j + 1];
          bad |= !(fabsf(a) <= 65504.f) || !(fabsf(b) <= 65504.f);
          __half2 h = __floats2half2_rn(a, b);
          pk[j] = *reinterpret_cast<uint32_t*>(&h);
          part += f[2 * j] * f[2 * j] + f[2 * j + 1] * f[2 * j + 1];
        }
        reinterpret_cast<uint4*>(xh + t * d)[c] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
      }
    }
    if (ss) {
      // lanes 16k .. 16k+15 hold columns [128 * (c0 / 16 + k), +128): reduce within the half-warp
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
      const int slot = (c0 * 8 + (lane >> 4) * 128) / 128;
      if ((lane & 15) == 0 && c < d / 8) ss[t * (d / 128) + slot] = part;
    }
  }
  if (bad) set_dev_error(err, DEVERR_FP16_RANGE);
}

// One warp per row: fp32 statistics, fp16 output for the next GEMM.
// split: out rows are 2d wide, fp16(v) in [0, d) and fp16(v - fp16(v)) in
// [d, 2d), a two-term operand for a GEMM that runs over K = 2d against the
// weight stored twice along K.
template <int PER_LANE>  // d / 32 / 4 float4 per lane (compile-time for register residency)
__global__ void k_rmsnorm(const float* x, int64_t T, int d, const uint16_t* g, float eps, __half* out, int split,
                          int* err) {
  const int64_t t = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (t >= T) return;
  const float4* row = reinterpret_cast<const float4*>(x + t * d);
  float4 v[PER_LANE];
  float ss = 0.f;
#pragma unroll
  for (int j = 0; j < PER_LANE; ++j) {
    v[j] = row[lane + 32 * j];
    ss += v[j].x * v[j].x + v[j].y * v[j].y + v[j].z * v[j].z + v[j].w * v[j].w;
  }
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / d + eps);
  bool bad = false;
  uint2* o = reinterpret_cast<uint2*>(out + t * d * (split ? 2 : 1));
  uint2* ol = reinterpret_cast<uint2*>(out + t * d * 2 + d);
#pragma unroll
  for (int j = 0; j < PER_LANE; ++j) {
    const int c = (lane + 32 * j) * 4;
    float g0 = 1.f, g1 = 1.f, g2 = 1.f, g3 = 1.f;
    if (g) {
      const uint2 gg = *reinterpret_cast<const uint2*>(g + c);
      g0 = __uint_as_float(gg.x << 16);
      g1 = __uint_as_float(gg.x & 0xFFFF0000u);
      g2 = __uint_as_float(gg.y << 16);
      g3 = __uint_as_float(gg.y & 0xFFFF0000u);
    }
    const float a = v[j].x * inv * g0, b = v[j].y * inv * g1, cc = v[j].z * inv * g2, e = v[j].w * inv * g3;
    bad |= !(fabsf(a) <= 65504.f) || !(fabsf(b) <= 65504.f) || !(fabsf(cc) <= 65504.f) || !(fabsf(e) <= 65504.f);
    __half2 h0 = __floats2half2_rn(a, b), h1 = __floats2half2_rn(cc, e);
    o[lane + 32 * j] = make_uint2(*reinterpret_cast<uint32_t*>(&h0), *reinterpret_cast<uint32_t*>(&h1));
    if (split) {
      const float2 f0 = __half22float2(h0), f1 = __half22float2(h1);
      __half2 l0 = __floats2half2_rn(a - f0.x, b - f0.y), l1 = __floats2half2_rn(cc - f1.x, e - f1.y);
      ol[lane + 32 * j] = make_uint2(*reinterpret_cast<uint32_t*>(&l0), *reinterpret_cast<uint32_t*>(&l1));
    }
  }
  if (bad) set_dev_error(err, DEVERR_FP16_RANGE);
}

// Generic-width fallback (d not a multiple of 128 handled elsewhere; d % 4 == 0 here).
__global__ void k_rmsnorm_any(const float* x, int64_t T, int d, const uint16_t* g, float eps, __half* out, int split,
                              int* err) {
  const int64_t t = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (t >= T) return;
  const float* row = x + t * d;
  float ss = 0.f;
  for (int c = lane; c < d; c += 32) ss += row[c] * row[c];
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / d + eps);
  bool bad = false;
  for (int c = lane; c < d; c += 32) {
    const float v = row[c] * inv * (g ? bf16_bits_to_float(g[c]) : 1.f);
    bad |= !(fabsf(v) <= 65504.f);
    const __half h = __float2half_rn(v);
    out[t * d * (split ? 2 : 1) + c] = h;
    if (split) out[t * d * 2 + d + c] = __float2half_rn(v - __half2float(h));
  }
  if (bad) set_dev_error(err, DEVERR_FP16_RANGE);
}

// One warp per candidate row: final RMSNorm of the last token's hidden state,
// then K dot products with the label rows of the LM head plus its bias.
__global__ void k_label_head(const float* resid, const int32_t* last_idx, const float* prefix_last, int64_t n, int d,
                             const uint16_t* g, float eps, const uint16_t* W, const uint16_t* bias,
                             const int32_t* labels, int K, float* logits) {
  const int64_t r = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (r >= n) return;
  const int32_t li = last_idx[r];
  const float* x = li >= 0 ? resid + static_cast<int64_t>(li) * d : prefix_last;
  float ss = 0.f;
  for (int c = lane; c < d; c += 32) ss += x[c] * x[c];
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / d + eps);
  for (int k = 0; k < K; ++k) {
    const uint16_t* w = W + static_cast<int64_t>(labels[k]) * d;
    float acc = 0.f;
    for (int c = lane; c < d; c += 32) acc += x[c] * inv * bf16_bits_to_float(g[c]) * bf16_bits_to_float(w[c]);
    acc = warp_sum(acc);
    if (lane == 0) logits[r * K + k] = acc + bf16_bits_to_float(bias[labels[k]]);
  }
}

// Final layer, rows only: gather each row's last token (attention output and
// residual) into dense [n, .] buffers; last_compact[r] = r, or -1 for a row
// without tokens of its own (its logits come from the prefix's last state).
__global__ void k_gather_last(const __half* att, int ld_att, const float* resid, int d, const int32_t* last_idx,
                              int64_t n, __half* att_out, float* resid_out, int32_t* last_compact) {
  const int64_t r = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (r >= n) return;
  const int32_t li = last_idx[r];
  if (lane == 0) last_compact[r] = li >= 0 ? static_cast<int32_t>(r) : -1;
  const int64_t src = li >= 0 ? li : 0;
  const uint4* a = reinterpret_cast<const uint4*>(att + src * ld_att);
  uint4* ao = reinterpret_cast<uint4*>(att_out + r * ld_att);
  for (int c = lane; c < ld_att / 8; c += 32) ao[c] = a[c];
  const float4* x = reinterpret_cast<const float4*>(resid + src * d);
  float4* xo = reinterpret_cast<float4*>(resid_out + r * d);
  for (int c = lane; c < d / 4; c += 32) xo[c] = x[c];
}

inline unsigned grid_for(int64_t threads) { return static_cast<unsigned>((threads + 255) / 256); }

}  // namespace

void launch_bf16_to_f16(const uint16_t* src, __half* dst, int64_t rows, int64_t cols, int interleave_block,
                        int64_t half_rows, int* err, cudaStream_t s, int64_t ldd) {
  const int64_t n = rows * cols;
  if (n <= 0) return;
  unsigned g = grid_for(n);
  if (g > 8192) g = 8192;
  k_bf16_to_f16<<<g, 256, 0, s>>>(src, dst, rows, cols, interleave_block, half_rows, ldd > 0 ? ldd : cols, err);
}

void launch_rope_table(float* cos_t, float* sin_t, int max_pos, int head_dim, float theta, cudaStream_t s) {
  const int64_t n = static_cast<int64_t>(max_pos) * (head_dim / 2);
  if (n <= 0) return;
  unsigned g = grid_for(n);
  if (g > 4096) g = 4096;
  k_rope_table<<<g, 256, 0, s>>>(cos_t, sin_t, max_pos, head_dim, static_cast<double>(theta));
}

void launch_embed(const int32_t* tok, int64_t T, const uint16_t* emb, int d, float* resid, __half* xh, float* ss,
                  const uint16_t* gain, int* err, cudaStream_t s) {
  if (T <= 0) return;
  k_embed<<<grid_for(T * 32), 256, 0, s>>>(tok, T, emb, d, resid, xh, ss, gain, err);
}

void launch_rmsnorm(const float* x, int64_t T, int d, const uint16_t* g, float eps, __half* out, int* err,
                    cudaStream_t s, bool split) {
  if (T <= 0) return;
  const unsigned grid = grid_for(T * 32);
  const int sp = split ? 1 : 0;
  switch (d) {
    case 128: k_rmsnorm<1><<<grid, 256, 0, s>>>(x, T, d, g, eps, out, sp, err); break;
    case 256: k_rmsnorm<2><<<grid, 256, 0, s>>>(x, T, d, g, eps, out, sp, err); break;
    case 512: k_rmsnorm<4><<<grid, 256, 0, s>>>(x, T, d, g, eps, out, sp, err); break;
    case 1024: k_rmsnorm<8><<<grid, 256, 0, s>>>(x, T, d, g, eps, out, sp, err); break;
    case 2048: k_rmsnorm<16><<<grid, 256, 0, s>>>(x, T, d, g, eps, out, sp, err); break;
    case 4096: k_rmsnorm<32><<<grid, 256, 0, s>>>(x, T, d, g, eps, out, sp, err); break;
    default: k_rmsnorm_any<<<grid, 256, 0, s>>>(x, T, d, g, eps, out, sp, err); break;
  }
}

void launch_gather_last(const __half* att, int ld_att, const float* resid, int d, const int32_t* last_idx, int64_t n,
                        __half* att_out, float* resid_out, int32_t* last_compact, cudaStream_t s) {
  if (n <= 0) return;
  k_gather_last<<<grid_for(n * 32), 256, 0, s>>>(att, ld_att, resid, d, last_idx, n, att_out, resid_out, last_compact);
}

void launch_label_head(const float* resid, const int32_t* last_idx, const float* prefix_last, int64_t n_rows, int d,
                       const uint16_t* g, float eps, const uint16_t* lm_head, const uint16_t* lm_bias,
                       const int32_t* labels, int n_labels, float* logits_out, cudaStream_t s) {
  if (n_rows <= 0) return;
  k_label_head<<<grid_for(n_rows * 32), 256, 0, s>>>(resid, last_idx, prefix_last, n_rows, d, g, eps, lm_head,
                                                     lm_bias, labels, n_labels, logits_out);
}

}  // namespace aiq
