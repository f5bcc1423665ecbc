// Prefill GEMM on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// C = A[M,K] * B[N,K]^T: A is the packed activation (tokens x features, fp16),
// B a linear layer's weight in [out, in] layout (fp16 copy of the bf16 model),
// accumulation in fp32 TMEM.  These are the decoder's dense contractions
// (QKV, O, gate/up and down projections of each layer) run over every token
// of the packed variable-length batch.
//
// Structure (one CTA per SM, persistent over 128 x BN output tiles, tiles
// ordered in bands of output columns so running CTAs share one L2-resident
// slice of the weight matrix):
//   warp 0  : TMA producer, STAGES-deep ring of (A 128x64, B BNx64) tiles,
//             128-byte swizzle, one mbarrier per stage (full / empty).
//   warp 1  : allocates 2*BN TMEM columns (two accumulators) and issues
//             tcgen05.mma 128xBNx16 from one thread; tcgen05.commit frees a
//             smem stage and, per tile, signals the epilogue.
//   warps 2-5: epilogue; each thread owns one accumulator row (TMEM lane),
//             reads 32-column slices with tcgen05.ld and applies the fused
//             epilogue (RoPE, SwiGLU, fp32 residual add) while the MMA warp
//             already fills the other accumulator.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"

namespace aiq {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;      // 64 fp16 = 128 bytes = one swizzle row
constexpr int UMMA_K = 16;  // K of one kind::f16 MMA
constexpr int kThreads = 192;

template <int BN>
struct Cfg {
  static constexpr int STAGES = BN == 256 ? 4 : 6;
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 2 * BN;  // double-buffered fp32 accumulator
  static constexpr int BAR_BYTES = 256;
  static constexpr int SMEM = 1024 /*align slack*/ + STAGES * STAGE_BYTES + BAR_BYTES;
};

struct KArgs {
  int M, N, K;
  GemmEpilogue ep;
};

// EPI_RESID_ADD stages the accumulator in shared memory for TMA reduce-add:
// per epilogue warp two 32 x 32 fp32 buffers (4 KB each, 128-byte swizzle),
// after the operand ring and the barriers, 1024-byte aligned.
template <int EPI>
constexpr int epi_stage_bytes() {
  return EPI == EPI_RESID_ADD ? 4 * 2 * 4096 : 0;
}
constexpr int round_up_1k(int x) { return (x + 1023) & ~1023; }

// Tile order: bands of at most kBandTiles output-tile columns, all row tiles
// of a band before the next band, columns fastest within a band.  Running
// CTAs then share one band of the weight matrix (<= 32 MB for 2048-deep K)
// that stays in L2 while the activation rows stream past, instead of sweeping
// the whole weight matrix once per row tile.
constexpr int kBandTiles = 32;

__device__ __forceinline__ void tile_coords(int tile, int num_m, int num_n, int& mt, int& nt) {
  const int bw = num_n < kBandTiles ? num_n : kBandTiles;
  const int full_bands = num_n / bw;
  const int per_band = num_m * bw;
  const int band = tile / per_band;
  if (band < full_bands) {
    const int r = tile - band * per_band;
    mt = r / bw;
    nt = band * bw + r % bw;
  } else {  // the narrower last band
    const int w = num_n - full_bands * bw;
    const int r = tile - full_bands * per_band;
    mt = r / w;
    nt = full_bands * bw + r % w;
  }
}

__device__ __forceinline__ float u2f(uint32_t u) { return __uint_as_float(u); }

__device__ __forceinline__ void store_f16x32(__half* dst, const float* v, bool& bad) {
  uint4 pk[4];
  uint32_t* w = reinterpret_cast<uint32_t*>(pk);
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const float a = v[2 * j], b = v[2 * j + 1];
    bad |= !(fabsf(a) <= 65504.f) || !(fabsf(b) <= 65504.f);
    __half2 h = __floats2half2_rn(a, b);
    w[j] = *reinterpret_cast<uint32_t*>(&h);
  }
  uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int j = 0; j < 4; ++j) d[j] = pk[j];
}

__device__ __forceinline__ void load32(uint32_t taddr, float* v) {
  uint32_t r[32];
  tmem_ld_32x32b_x32(taddr, r);
  tmem_ld_wait();
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = u2f(r[j]);
}

// Two 32-column slices with one wait (both loads in flight together).
__device__ __forceinline__ void load2x32(uint32_t ta, uint32_t tb, float* va, float* vb) {
  uint32_t ra[32], rb[32];
  tmem_ld_32x32b_x32(ta, ra);
  tmem_ld_32x32b_x32(tb, rb);
  tmem_ld_wait();
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    va[j] = u2f(ra[j]);
    vb[j] = u2f(rb[j]);
  }
}

__device__ __forceinline__ void load_f32x32(const float* src, float* v) {
  const float4* p = reinterpret_cast<const float4*>(src);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const float4 x = __ldg(p + j);
    v[4 * j] = x.x;
    v[4 * j + 1] = x.y;
    v[4 * j + 2] = x.z;
    v[4 * j + 3] = x.w;
  }
}

// dst += v (fp32), and the new values are returned in out.
__device__ __forceinline__ void add_store_f32x32(float* dst, const float* v, float* out) {
  float4* p = reinterpret_cast<float4*>(dst);
  float4 x[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) x[j] = p[j];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    x[j].x += v[4 * j];
    x[j].y += v[4 * j + 1];
    x[j].z += v[4 * j + 2];
    x[j].w += v[4 * j + 3];
    p[j] = x[j];
    out[4 * j] = x[j].x;
    out[4 * j + 1] = x[j].y;
    out[4 * j + 2] = x[j].z;
    out[4 * j + 3] = x[j].w;
  }
}

// 1 / RMS of an accumulator row from its partial sums of squares (fixed
// summation order), or 1 when the GEMM's input is already normalised.
__device__ __forceinline__ float row_inv_rms(const GemmEpilogue& ep, int row, bool live) {
  if (!ep.row_ss || !live) return 1.f;
  const float* p = ep.row_ss + static_cast<int64_t>(row) * ep.ss_parts;
  float s = 0.f;
  if ((ep.ss_parts & 3) == 0) {
    const float4* p4 = reinterpret_cast<const float4*>(p);
    for (int i = 0; i < ep.ss_parts / 4; ++i) {
      const float4 v = __ldg(p4 + i);
      s += v.x;
      s += v.y;
      s += v.z;
      s += v.w;
    }
  } else {
    for (int i = 0; i < ep.ss_parts; ++i) s += p[i];
  }
  return rsqrtf(s / ep.d_norm + ep.eps);
}

__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// Issued before the epilogue waits for its accumulator: pulls the bytes this
// thread's row will read into L2 while the tile's MMAs still run.
template <int BN, int EPI>
__device__ __forceinline__ void epilogue_prefetch(const KArgs& a, int row, int n0) {
  if (row >= a.M) return;
  const GemmEpilogue& ep = a.ep;
  if constexpr (EPI == EPI_RESID_F32) {
    prefetch_l2(static_cast<const float*>(ep.out) + static_cast<int64_t>(row) * ep.ldo + n0, BN * 4);
  } else if constexpr (EPI == EPI_ROPE_F16) {
    if (n0 < ep.rope_cols) {
      const int half = ep.head_dim >> 1;
      const int64_t off = static_cast<int64_t>(ep.positions[row]) * half;
      prefetch_l2(ep.rope_cos + off, half * 4);
      prefetch_l2(ep.rope_sin + off, half * 4);
    }
  }
}

// inv: the row's 1/RMS (fused RMSNorm), computed by the caller before it
// waits for the accumulator, so that its loads overlap the tile's MMAs.
template <int BN, int EPI>
__device__ __forceinline__ void epilogue_tile(const KArgs& a, uint32_t trow, int row, int n0, float inv) {
  const GemmEpilogue& ep = a.ep;
  const bool live = row < a.M;
  bool bad = false;
  if constexpr (EPI == EPI_RESID_F32) {
    float* o = static_cast<float*>(ep.out) + static_cast<int64_t>(row) * ep.ldo + n0;
    float part = 0.f;  // sum of squares of the new residual over 128 columns
#pragma unroll 1
    for (int c = 0; c < BN; c += 64) {
      float v0[32], v1[32];
      load2x32(trow + c, trow + c + 32, v0, v1);
      if (live) {
        add_store_f32x32(o + c, v0, v0);
        add_store_f32x32(o + c + 32, v1, v1);
        if (ep.xh_out) {
          __half* xh = ep.xh_out + static_cast<int64_t>(row) * ep.ldo + n0 + c;
#pragma unroll
          for (int j = 0; j < 32; ++j) part += v0[j] * v0[j] + v1[j] * v1[j];
          if (ep.xh_gain) {
            // the next attention norm's gain goes on the activation (the QKV
            // weights stay exact): one fp16 rounding of x * g per element
            const uint4* g4 = reinterpret_cast<const uint4*>(ep.xh_gain + n0 + c);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const uint4 gv = __ldg(g4 + q);
              const uint32_t gw[4] = {gv.x, gv.y, gv.z, gv.w};
              float* v = q < 4 ? v0 + 8 * q : v1 + 8 * (q - 4);
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                v[2 * j] *= __uint_as_float(gw[j] << 16);
                v[2 * j + 1] *= __uint_as_float(gw[j] & 0xFFFF0000u);
              }
            }
          }
          store_f16x32(xh, v0, bad);
          store_f16x32(xh + 32, v1, bad);
          if ((c & 127) == 64) {
            ep.ss_out[static_cast<int64_t>(row) * ep.ss_parts + (n0 + c) / 128] = part;
            part = 0.f;
          }
        }
      }
    }
  } else if constexpr (EPI == EPI_ARGMAX) {
    // logits = acc + bias; strictly-greater keeps the first column of a tie
    float best = -INFINITY;
    int bcol = -1;
#pragma unroll 1
    for (int c = 0; c < BN; c += 64) {
      float v0[32], v1[32];
      load2x32(trow + c, trow + c + 32, v0, v1);
      if (live) {
        float b0[32], b1[32];
        load_f32x32(ep.bias + n0 + c, b0);
        load_f32x32(ep.bias + n0 + c + 32, b1);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const float x = v0[j] + b0[j];
          if (x > best) {
            best = x;
            bcol = n0 + c + j;
          }
        }
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const float x = v1[j] + b1[j];
          if (x > best) {
            best = x;
            bcol = n0 + c + 32 + j;
          }
        }
      }
    }
    if (live && bcol >= 0) {
      const uint32_t u = __float_as_uint(best);
      const uint32_t ord = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
      atomicMax(ep.best + row,
                (static_cast<unsigned long long>(ord) << 32) | (0xFFFFFFFFu - static_cast<uint32_t>(bcol)));
    }
  } else if constexpr (EPI == EPI_SWIGLU_F16) {
    __half* o = static_cast<__half*>(ep.out) + static_cast<int64_t>(row) * ep.ldo + n0 / 2;
#pragma unroll 1
    for (int c = 0; c < BN / 2; c += 32) {
      float g[32], u[32];
      load2x32(trow + c, trow + BN / 2 + c, g, u);
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const float gj = g[j] * inv;
        g[j] = gj / (1.0f + expf(-gj)) * (u[j] * inv);
      }
      if (live) {
        store_f16x32(o + c, g, bad);
        if (ep.lo_off > 0) {
#pragma unroll
          for (int j = 0; j < 32; ++j) u[j] = g[j] - __half2float(__float2half_rn(g[j]));
          store_f16x32(o + ep.lo_off + c, u, bad);
        }
      }
    }
  } else {
    __half* o = static_cast<__half*>(ep.out) + static_cast<int64_t>(row) * ep.ldo + n0;
    int rot_end = 0;  // columns [0, rot_end) of the tile hold rotated (q, k) heads
    if constexpr (EPI == EPI_ROPE_F16) {
      const int hd = ep.head_dim;
      const int half = hd >> 1;
      rot_end = ep.rope_cols - n0;
      rot_end = rot_end < 0 ? 0 : (rot_end > BN ? BN : rot_end);
      const int64_t toff = live ? static_cast<int64_t>(ep.positions[row]) * half : 0;
      if (half >= 32) {
        // cos/sin of this row's position, 32 frequencies at a time, reused by every head of the tile
#pragma unroll 1
        for (int i0 = 0; i0 < half; i0 += 32) {
          float cs[32], sn[32];
          load_f32x32(ep.rope_cos + toff + i0, cs);
          load_f32x32(ep.rope_sin + toff + i0, sn);
#pragma unroll 1
          for (int h = 0; h < rot_end; h += hd) {
            float x1[32], x2[32];
            load2x32(trow + h + i0, trow + h + half + i0, x1, x2);
            if (live) {
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                const float a1 = x1[j] * inv, a2 = x2[j] * inv;
                x1[j] = a1 * cs[j] - a2 * sn[j];
                x2[j] = a2 * cs[j] + a1 * sn[j];
              }
              store_f16x32(o + h + i0, x1, bad);
              store_f16x32(o + h + half + i0, x2, bad);
            }
          }
        }
      } else {  // head_dim 32: both halves of a head in one 32-column slice
        float cs[16], sn[16];
        const float4* c4 = reinterpret_cast<const float4*>(ep.rope_cos + toff);
        const float4* s4 = reinterpret_cast<const float4*>(ep.rope_sin + toff);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float4 cv = __ldg(c4 + j), sv = __ldg(s4 + j);
          cs[4 * j] = cv.x; cs[4 * j + 1] = cv.y; cs[4 * j + 2] = cv.z; cs[4 * j + 3] = cv.w;
          sn[4 * j] = sv.x; sn[4 * j + 1] = sv.y; sn[4 * j + 2] = sv.z; sn[4 * j + 3] = sv.w;
        }
#pragma unroll 1
        for (int h = 0; h < rot_end; h += 32) {
          float x[32];
          load32(trow + h, x);
          if (live) {
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const float a1 = x[j] * inv, a2 = x[j + 16] * inv;
              x[j] = a1 * cs[j] - a2 * sn[j];
              x[j + 16] = a2 * cs[j] + a1 * sn[j];
            }
            store_f16x32(o + h, x, bad);
          }
        }
      }
    }
    // plain fp16 columns (all of them for EPI_F16; the value heads for EPI_ROPE_F16)
    int c = rot_end;
#pragma unroll 1
    for (; c + 64 <= BN; c += 64) {
      float v0[32], v1[32];
      load2x32(trow + c, trow + c + 32, v0, v1);
      if (live) {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          v0[j] *= inv;
          v1[j] *= inv;
        }
        store_f16x32(o + c, v0, bad);
        store_f16x32(o + c + 32, v1, bad);
      }
    }
    if (c < BN) {
      float v[32];
      load32(trow + c, v);
      if (live) {
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] *= inv;
        store_f16x32(o + c, v, bad);
      }
    }
  }
  if (bad) set_dev_error(ep.err, DEVERR_FP16_RANGE);
}

__device__ __forceinline__ void st_shared_v4(uint32_t saddr, uint4 v) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(saddr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

// out[rows m0q .. m0q + 31][n0 .. n0 + BN) += acc, one 32 x 32 tile at a time:
// each lane writes its row (TMEM lane) into a swizzled staging buffer, lane 0
// hands the tile to the TMA unit as a reduce-add (rows past M are clipped by
// the tensor map).  Two buffers alternate; a buffer is rewritten only after
// the reduce issued from it two tiles earlier has read it.
template <int BN>
__device__ __forceinline__ void epilogue_tma_add(const CUtensorMap* tma_c, uint32_t trow, int m0q, int n0,
                                                 uint8_t* stage, int lane, uint32_t& nbuf) {
#pragma unroll 1
  for (int c = 0; c < BN; c += 32) {
    float v[32];
    load32(trow + c, v);
    uint8_t* buf = stage + (nbuf & 1) * 4096;
    if (lane == 0) bulk_wait_group_read<1>();
    __syncwarp();
    const uint32_t row = smem_u32(buf) + lane * 128;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      st_shared_v4(row + ((j ^ (lane & 7)) << 4), make_uint4(__float_as_uint(v[4 * j]), __float_as_uint(v[4 * j + 1]),
                                                             __float_as_uint(v[4 * j + 2]),
                                                             __float_as_uint(v[4 * j + 3])));
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_reduce_add_2d(tma_c, buf, n0 + c, m0q);
      bulk_commit_group();
    }
    ++nbuf;
  }
}

template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    k_gemm_tcgen05(const __grid_constant__ CUtensorMap tma_a, const __grid_constant__ CUtensorMap tma_b,
                   const __grid_constant__ CUtensorMap tma_c, KArgs args) {
  using C = Cfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + C::STAGES;
  uint64_t* tfull = bars + 2 * C::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  int* err = args.ep.err;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 4);  // one arrival per epilogue warp
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tma_a);
    tma_prefetch_desc(&tma_b);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int num_n = args.N / BN;
  const int num_m = (args.M + BM - 1) / BM;
  const int num_tiles = num_m * num_n;
  const int kblocks = args.K / BK;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------- TMA producer
      uint32_t issued = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        int mt, nt;
        tile_coords(tile, num_m, num_n, mt, nt);
        const int m0 = mt * BM;
        const int n0 = nt * BN;
        for (int kb = 0; kb < kblocks; ++kb) {
          const int s = issued % C::STAGES;
          const uint32_t ph = (issued / C::STAGES) & 1;
          if (!mbar_wait_bounded(&empty[s], ph ^ 1, abort_flag, err)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], C::STAGE_BYTES);
          tma_load_2d(sA + s * C::A_BYTES, &tma_a, &full[s], kb * BK, m0);
          tma_load_2d(sB + s * C::B_BYTES, &tma_b, &full[s], kb * BK, n0);
          ++issued;
        }
      }
      if (!ok) {
        // drain this thread's copies still in flight before the CTA can exit
        const uint32_t first = issued > (uint32_t)C::STAGES ? issued - C::STAGES : 0;
        volatile int never = 0;
        for (uint32_t i = first; i < issued; ++i)
          mbar_wait_bounded(&full[i % C::STAGES], (i / C::STAGES) & 1, &never, nullptr, 200000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------ MMA issuer
      constexpr uint32_t idesc = idesc_f16_f32(BM, BN);
      uint32_t consumed = 0;
      int acc = 0;
      uint32_t acc_ph = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        if (!mbar_wait_bounded(&tempty[acc], acc_ph ^ 1, abort_flag, err)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = 0; kb < kblocks; ++kb) {
          const int s = consumed % C::STAGES;
          const uint32_t ph = (consumed / C::STAGES) & 1;
          if (!mbar_wait_bounded(&full[s], ph, abort_flag, err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + s * C::A_BYTES);
          const uint32_t b0 = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / UMMA_K; ++k) {
            // advancing K inside the 128-byte swizzle row = +32 bytes on the start address
            umma_f16_ss(d_tmem, smem_desc_k_sw128(a0 + k * UMMA_K * 2), smem_desc_k_sw128(b0 + k * UMMA_K * 2),
                        idesc, (kb | k) != 0);
          }
          umma_commit(&empty[s]);
          ++consumed;
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
        acc ^= 1;
        if (acc == 0) acc_ph ^= 1;
      }
      // every MMA issued above has completed once this arrives
      umma_commit(mma_done);
      volatile int never = 0;
      mbar_wait_bounded(mma_done, 0, &never, err);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quarter = warp & 3;  // TMEM lanes this warp may access
    uint8_t* stage = smem + round_up_1k(C::STAGES * C::STAGE_BYTES + C::BAR_BYTES) + quarter * 8192;
    uint32_t nbuf = 0;
    int acc = 0;
    uint32_t acc_ph = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
      int mt, nt;
      tile_coords(tile, num_m, num_n, mt, nt);
      const int m0 = mt * BM;
      const int n0 = nt * BN;
      epilogue_prefetch<BN, EPI>(args, m0 + quarter * 32 + lane, n0);
      const float inv = (EPI == EPI_ROPE_F16 || EPI == EPI_SWIGLU_F16)
                            ? row_inv_rms(args.ep, m0 + quarter * 32 + lane, m0 + quarter * 32 + lane < args.M)
                            : 1.f;
      // warp-uniform: a lane that gives up makes the whole warp give up, so no
      // lane is left alone in the warp-synchronous TMEM loads of the epilogue
      if (!__all_sync(0xffffffffu, mbar_wait_bounded(&tfull[acc], acc_ph, abort_flag, err))) break;
      tc_fence_after();
      const uint32_t trow = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
      if constexpr (EPI == EPI_RESID_ADD)
        epilogue_tma_add<BN>(&tma_c, trow, m0 + quarter * 32, n0, stage, lane, nbuf);
      else
        epilogue_tile<BN, EPI>(args, trow, m0 + quarter * 32 + lane, n0, inv);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
      acc ^= 1;
      if (acc == 0) acc_ph ^= 1;
    }
    if constexpr (EPI == EPI_RESID_ADD) {
      if (lane == 0) bulk_wait_group_all();  // the reduces have completed before the CTA leaves
    }
  }

  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}


// ------------------------------------------------------------ CTA pairs ---
// 256 x 256 output tiles on a cluster of two CTAs (tcgen05.mma.cta_group::2).
// Each CTA stages its own 128 rows of A and 128 columns of B per 128-deep
// k-block (two 64-deep swizzled sub-blocks per operand, 64 KB, 3 stages), so
// every SM moves half the B bytes of the single-CTA 128 x 256 tile for the
// same MMA work, and each barrier wait, fence and commit of the MMA issuer
// covers eight MMAs instead of four (3-6 % faster than 64-deep stages on the
// QKV and gate/up shapes); its TMA completes on the leader's barrier, the
// leader alone issues the M = 256 MMA, and each CTA's epilogue drains its own
// 128 accumulator rows and reports back to the leader.  Needs K % 128 == 0
// (other K take the single-CTA kernel).
struct CfgPair {
  static constexpr int STAGES = 3;
  static constexpr int SUB = 2;                  // 64-deep sub-blocks per stage
  static constexpr int A_BYTES = SUB * 128 * BK * 2;
  static constexpr int B_BYTES = SUB * 128 * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = 512;
  static constexpr int SMEM = 1024 + STAGES * STAGE_BYTES + 256;
};

template <int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    k_gemm_tcgen05_pair(const __grid_constant__ CUtensorMap tma_a, const __grid_constant__ CUtensorMap tma_b,
                        const __grid_constant__ CUtensorMap tma_c, KArgs args) {
  using C = CfgPair;
  constexpr int BN = 256;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES);
  uint64_t* full = bars;                 // used in the leader only
  uint64_t* empty = bars + C::STAGES;    // per CTA, multicast by the leader's commits
  uint64_t* tfull = bars + 2 * C::STAGES;
  uint64_t* tempty = tfull + 2;          // used in the leader only: 4 warps x 2 CTAs
  uint64_t* mma_done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int pair = blockIdx.x >> 1;
  const int n_pairs = gridDim.x >> 1;
  int* err = args.ep.err;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 8);
    }
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tma_a);
    tma_prefetch_desc(&tma_b);
  }
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, C::TMEM_COLS);
    tmem_relinquish_pair();
    tc_fence_before();
  }
  __syncthreads();
  cluster_sync();  // barriers of both CTAs initialised before any remote arrival
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int num_n = args.N / BN;
  const int num_m = (args.M + 2 * BM - 1) / (2 * BM);
  const int num_tiles = num_m * num_n;
  const int kblocks = args.K / (BK * C::SUB);

  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------- TMA producer
      const uint32_t full_leader = map_to_cta(smem_u32(full), 0);
      uint32_t issued = 0;
      bool ok = true;
      for (int tile = pair; tile < num_tiles && ok; tile += n_pairs) {
        int mt, nt;
        tile_coords(tile, num_m, num_n, mt, nt);
        const int m0 = mt * 2 * BM;
        const int n0 = nt * BN;
        for (int kb = 0; kb < kblocks; ++kb) {
          const int s = issued % C::STAGES;
          const uint32_t ph = (issued / C::STAGES) & 1;
          if (!mbar_wait_bounded(&empty[s], ph ^ 1, abort_flag, err)) {
            ok = false;
            break;
          }
          if (leader) mbar_arrive_expect_tx(&full[s], 2 * C::STAGE_BYTES);
#pragma unroll
          for (int sb = 0; sb < C::SUB; ++sb) {
            tma_load_2d_pair(sA + s * C::A_BYTES + sb * (128 * BK * 2), &tma_a, full_leader + s * 8,
                             (kb * C::SUB + sb) * BK, m0 + rank * BM);
            tma_load_2d_pair(sB + s * C::B_BYTES + sb * (128 * BK * 2), &tma_b, full_leader + s * 8,
                             (kb * C::SUB + sb) * BK, n0 + rank * 128);
          }
          ++issued;
        }
      }
      if (!ok && leader) {
        // the leader's barrier completes only once both CTAs' bytes have landed
        const uint32_t first = issued > (uint32_t)C::STAGES ? issued - C::STAGES : 0;
        volatile int never = 0;
        for (uint32_t i = first; i < issued; ++i)
          mbar_wait_bounded(&full[i % C::STAGES], (i / C::STAGES) & 1, &never, nullptr, 200000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ------------------------------------------------ MMA issuer (leader)
      constexpr uint32_t idesc = idesc_f16_f32(2 * BM, BN);
      uint32_t consumed = 0;
      int acc = 0;
      uint32_t acc_ph = 0;
      bool ok = true;
      for (int tile = pair; tile < num_tiles && ok; tile += n_pairs) {
        if (!mbar_wait_bounded(&tempty[acc], acc_ph ^ 1, abort_flag, err)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        for (int kb = 0; kb < kblocks; ++kb) {
          const int s = consumed % C::STAGES;
          const uint32_t ph = (consumed / C::STAGES) & 1;
          if (!mbar_wait_bounded(&full[s], ph, abort_flag, err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + s * C::A_BYTES);
          const uint32_t b0 = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
          for (int sb = 0; sb < C::SUB; ++sb)
#pragma unroll
            for (int k = 0; k < BK / UMMA_K; ++k)
              umma_f16_ss_pair(d_tmem, smem_desc_k_sw128(a0 + sb * (128 * BK * 2) + k * UMMA_K * 2),
                               smem_desc_k_sw128(b0 + sb * (128 * BK * 2) + k * UMMA_K * 2), idesc,
                               (kb | sb | k) != 0);
          umma_commit_pair_mc(&empty[s], 0x3);
          ++consumed;
        }
        if (!ok) break;
        umma_commit_pair_mc(&tfull[acc], 0x3);
        acc ^= 1;
        if (acc == 0) acc_ph ^= 1;
      }
      umma_commit_pair_mc(mma_done, 0x1);
      volatile int never = 0;
      mbar_wait_bounded(mma_done, 0, &never, err);
    }
  } else {
    // ------------------------------------------------ epilogue (both CTAs)
    const int quarter = warp & 3;
    const uint32_t tempty_leader = map_to_cta(smem_u32(tempty), 0);
    uint8_t* stage = smem + round_up_1k(C::STAGES * C::STAGE_BYTES + 256) + quarter * 8192;
    uint32_t nbuf = 0;
    int acc = 0;
    uint32_t acc_ph = 0;
    for (int tile = pair; tile < num_tiles; tile += n_pairs) {
      int mt, nt;
      tile_coords(tile, num_m, num_n, mt, nt);
      const int m0 = mt * 2 * BM + rank * BM;
      const int n0 = nt * BN;
      epilogue_prefetch<BN, EPI>(args, m0 + quarter * 32 + lane, n0);
      const float inv = (EPI == EPI_ROPE_F16 || EPI == EPI_SWIGLU_F16)
                            ? row_inv_rms(args.ep, m0 + quarter * 32 + lane, m0 + quarter * 32 + lane < args.M)
                            : 1.f;
      // warp-uniform: a lane that gives up makes the whole warp give up, so no
      // lane is left alone in the warp-synchronous TMEM loads of the epilogue
      if (!__all_sync(0xffffffffu, mbar_wait_bounded(&tfull[acc], acc_ph, abort_flag, err))) break;
      tc_fence_after();
      const uint32_t trow = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + acc * BN;
      if constexpr (EPI == EPI_RESID_ADD)
        epilogue_tma_add<BN>(&tma_c, trow, m0 + quarter * 32, n0, stage, lane, nbuf);
      else
        epilogue_tile<BN, EPI>(args, trow, m0 + quarter * 32 + lane, n0, inv);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(tempty_leader + acc * 8);
      acc ^= 1;
      if (acc == 0) acc_ph ^= 1;
    }
    if constexpr (EPI == EPI_RESID_ADD) {
      if (lane == 0) bulk_wait_group_all();  // the reduces have completed before the CTA leaves
    }
  }

  __syncthreads();
  cluster_sync();  // no CTA leaves while its peer may still signal it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, C::TMEM_COLS);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D fp16 tensor [rows, cols] (cols contiguous, row pitch ld elements), box 64 x box_rows, 128B swizzle.
bool make_map(CUtensorMap* m, const __half* base, int64_t rows, int64_t cols, int64_t ld, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld * 2)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<__half*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 2-D fp32 tensor [rows, cols] (row pitch ld elements), box 32 x 32, 128B swizzle:
// the target of EPI_RESID_ADD's reduce-add tiles.
bool make_map_out_f32(CUtensorMap* m, float* base, int64_t rows, int64_t cols, int64_t ld) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld * 4)};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int BN, int EPI>
constexpr int smem_single() {
  using C = Cfg<BN>;
  return EPI == EPI_RESID_ADD ? 1024 + round_up_1k(C::STAGES * C::STAGE_BYTES + C::BAR_BYTES) + epi_stage_bytes<EPI>()
                              : C::SMEM;
}
template <int EPI>
constexpr int smem_pair() {
  using C = CfgPair;
  return EPI == EPI_RESID_ADD ? 1024 + round_up_1k(C::STAGES * C::STAGE_BYTES + 256) + epi_stage_bytes<EPI>()
                              : C::SMEM;
}
static_assert(smem_single<256, EPI_RESID_ADD>() <= 232448 && smem_single<128, EPI_RESID_ADD>() <= 232448 &&
                  smem_pair<EPI_RESID_ADD>() <= 232448,
              "shared memory per block");

template <int BN, int EPI>
int launch(const CUtensorMap& ma, const CUtensorMap& mb, const CUtensorMap& mc, const KArgs& a, int num_sms,
           cudaStream_t stream) {
  constexpr int SM = smem_single<BN, EPI>();
  cudaError_t e = cudaFuncSetAttribute(k_gemm_tcgen05<BN, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, SM);
  if (e != cudaSuccess) return e;
  const int tiles = ((a.M + BM - 1) / BM) * (a.N / BN);
  const int grid = tiles < num_sms ? tiles : num_sms;
  k_gemm_tcgen05<BN, EPI><<<grid, kThreads, SM, stream>>>(ma, mb, mc, a);
  return cudaGetLastError();
}

template <int EPI>
int launch_pair(const CUtensorMap& ma, const CUtensorMap& mb, const CUtensorMap& mc, const KArgs& a, int num_sms,
                cudaStream_t stream) {
  constexpr int SM = smem_pair<EPI>();
  cudaError_t e = cudaFuncSetAttribute(k_gemm_tcgen05_pair<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, SM);
  if (e != cudaSuccess) return e;
  const int tiles = ((a.M + 2 * BM - 1) / (2 * BM)) * (a.N / 256);
  const int pairs = tiles < num_sms / 2 ? tiles : num_sms / 2;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * pairs, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = SM;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, k_gemm_tcgen05_pair<EPI>, ma, mb, mc, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

int dispatch_pair(const CUtensorMap& ma, const CUtensorMap& mb, const CUtensorMap& mc, const KArgs& a, int num_sms,
                  cudaStream_t s) {
  switch (a.ep.kind) {
    case EPI_F16: return launch_pair<EPI_F16>(ma, mb, mc, a, num_sms, s);
    case EPI_ROPE_F16: return launch_pair<EPI_ROPE_F16>(ma, mb, mc, a, num_sms, s);
    case EPI_RESID_F32: return launch_pair<EPI_RESID_F32>(ma, mb, mc, a, num_sms, s);
    case EPI_SWIGLU_F16: return launch_pair<EPI_SWIGLU_F16>(ma, mb, mc, a, num_sms, s);
    case EPI_ARGMAX: return launch_pair<EPI_ARGMAX>(ma, mb, mc, a, num_sms, s);
    case EPI_RESID_ADD: return launch_pair<EPI_RESID_ADD>(ma, mb, mc, a, num_sms, s);
  }
  return cudaErrorInvalidValue;
}

template <int BN>
int dispatch_epi(const CUtensorMap& ma, const CUtensorMap& mb, const CUtensorMap& mc, const KArgs& a, int num_sms,
                 cudaStream_t s) {
  switch (a.ep.kind) {
    case EPI_F16: return launch<BN, EPI_F16>(ma, mb, mc, a, num_sms, s);
    case EPI_ROPE_F16: return launch<BN, EPI_ROPE_F16>(ma, mb, mc, a, num_sms, s);
    case EPI_RESID_F32: return launch<BN, EPI_RESID_F32>(ma, mb, mc, a, num_sms, s);
    case EPI_SWIGLU_F16: return launch<BN, EPI_SWIGLU_F16>(ma, mb, mc, a, num_sms, s);
    case EPI_ARGMAX: return launch<BN, EPI_ARGMAX>(ma, mb, mc, a, num_sms, s);
    case EPI_RESID_ADD: return launch<BN, EPI_RESID_ADD>(ma, mb, mc, a, num_sms, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

int gemm_f16_tcgen05(const __half* A, int64_t lda, const __half* B, int64_t ldb, int M, int N, int K, int bn,
                     bool pair, const GemmEpilogue& ep, int num_sms, cudaStream_t stream) {
  if (M == 0) return 0;
  if (M < 0 || N <= 0 || K <= 0 || K % BK != 0 || (bn != 128 && bn != 256) || N % bn != 0) return cudaErrorInvalidValue;
  if (pair && bn != 256) return cudaErrorInvalidValue;
  if (K % (BK * CfgPair::SUB) != 0) pair = false;  // CTA-pair stages hold 128-deep k-blocks
  if ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(B)) & 15) return cudaErrorMisalignedAddress;
  if ((lda * 2) % 16 != 0 || (ldb * 2) % 16 != 0) return cudaErrorInvalidValue;
  if (ep.kind == EPI_ROPE_F16) {
    const int hd = ep.head_dim;
    if (!(hd == 32 || hd == 64 || hd == 128) || bn % hd != 0 || !ep.positions || !ep.rope_cos) return cudaErrorInvalidValue;
  }
  if (ep.kind == EPI_ARGMAX && (!ep.bias || !ep.best)) return cudaErrorInvalidValue;
  if (ep.kind == EPI_RESID_ADD &&
      (!ep.out || (reinterpret_cast<uintptr_t>(ep.out) & 15) || (ep.ldo * 4) % 16 != 0 || ep.xh_out))
    return cudaErrorInvalidValue;
  CUtensorMap ma, mb, mc;
  if (!make_map(&ma, A, M, K, lda, BM) || !make_map(&mb, B, N, K, ldb, pair ? 128 : bn)) return cudaErrorInvalidValue;
  if (ep.kind == EPI_RESID_ADD) {
    if (!make_map_out_f32(&mc, static_cast<float*>(ep.out), M, N, ep.ldo)) return cudaErrorInvalidValue;
  } else {
    mc = ma;  // unused by the other epilogues
  }
  KArgs a{M, N, K, ep};
  if (pair) return dispatch_pair(ma, mb, mc, a, num_sms, stream);
  return bn == 256 ? dispatch_epi<256>(ma, mb, mc, a, num_sms, stream)
                   : dispatch_epi<128>(ma, mb, mc, a, num_sms, stream);
}

}  // namespace aiq
