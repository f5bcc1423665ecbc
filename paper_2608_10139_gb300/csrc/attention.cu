// Causal grouped-query attention over the packed variable-length batch.
//
// Each CTA computes one 64-row query block of one sequence for one query
// head; it walks the key/value blocks of the shared prompt prefix (computed
// once per query, keys/values in prefix_kv) and then those of its own
// sequence up to the block's last query (attention never crosses a row
// boundary of the batch; every prefix position precedes every row token), with an
// fp32 online softmax (running max and sum per query row) so the score matrix
// is never materialised.  K/V blocks are double-buffered in shared memory with
// cp.async; QK^T and PV run on m16n8k16 fp16 tensor-core MMAs with fp32
// accumulation.  Query head h reads key/value head h / (Hq / Hkv).
#include "common.cuh"
#include "kernels.h"

namespace aiq {
namespace {

constexpr int BQ = 64;
constexpr int BKV = 64;
constexpr int kThreads = 128;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(smem)), "l"(gmem), "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_h2(float a, float b) {
  __half2 h = __floats2half2_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

template <int HD>
__device__ __forceinline__ void load_rows(__half* dst, const __half* src, int row0, int nvalid, int64_t ld) {
  constexpr int LDS = HD + 8;
  constexpr int CH = HD / 8;  // 16-byte chunks per row
  for (int c = threadIdx.x; c < 64 * CH; c += kThreads) {
    const int r = c / CH, k = c - r * CH;
    const bool v = row0 + r < nvalid;
    const __half* s = src + static_cast<int64_t>(v ? row0 + r : 0) * ld + k * 8;
    cp_async16(dst + r * LDS + k * 8, s, v);
  }
}

template <int HD>
__global__ void __launch_bounds__(kThreads) k_attention(const __half* __restrict__ qkv, const int32_t* seq_start,
                                                        const int32_t* tile_seq, const int32_t* tile_q0,
                                                        const int32_t* n_tiles, int Hq, int Hkv,
                                                        const __half* __restrict__ prefix_kv, int P, float scale_log2,
                                                        __half* __restrict__ out) {
  constexpr int LDS = HD + 8;
  constexpr int KS = HD / 16;  // k-steps of QK^T
  constexpr int DN = HD / 8;   // 8-wide output column tiles
  extern __shared__ __align__(16) uint8_t smem_raw[];
  __half* sQ = reinterpret_cast<__half*>(smem_raw);
  __half* sK = sQ + BQ * LDS;     // [2][BKV][LDS]
  __half* sV = sK + 2 * BKV * LDS;

  const int tile = blockIdx.x;
  if (tile >= *n_tiles) return;
  const int h = blockIdx.y;
  const int kvh = h / (Hq / Hkv);
  const int s = tile_seq[tile];
  const int q0 = tile_q0[tile];
  const int st = seq_start[s];
  const int len = seq_start[s + 1] - st;
  const int64_t ld = static_cast<int64_t>(Hq + 2 * Hkv) * HD;
  const __half* Qg = qkv + static_cast<int64_t>(st) * ld + h * HD;
  const __half* Kg = qkv + static_cast<int64_t>(st) * ld + (Hq + kvh) * HD;
  const __half* Vg = qkv + static_cast<int64_t>(st) * ld + (Hq + Hkv + kvh) * HD;
  const int q_end = min(q0 + BQ, len);
  const int n_pre = (P + BKV - 1) / BKV;  // blocks of prefix keys (positions 0..P-1)
  const int n_kv = n_pre + (q_end + BKV - 1) / BKV;
  const int64_t ldp = static_cast<int64_t>(2 * Hkv) * HD;
  const __half* Kp = prefix_kv + kvh * HD;
  const __half* Vp = prefix_kv + (Hkv + kvh) * HD;
  auto load_kv = [&](int j, int buf) {
    if (j < n_pre) {
      load_rows<HD>(sK + buf * BKV * LDS, Kp, j * BKV, P, ldp);
      load_rows<HD>(sV + buf * BKV * LDS, Vp, j * BKV, P, ldp);
    } else {
      load_rows<HD>(sK + buf * BKV * LDS, Kg, (j - n_pre) * BKV, len, ld);
      load_rows<HD>(sV + buf * BKV * LDS, Vg, (j - n_pre) * BKV, len, ld);
    }
  };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gq = lane >> 2, tq = lane & 3;
  const int wrow0 = q0 + warp * 16;  // first query row of this warp (sequence-local)

  load_rows<HD>(sQ, Qg, q0, len, ld);
  load_kv(0, 0);
  cp_async_commit();

  uint32_t qf[KS][4];
  float o[DN][4];
#pragma unroll
  for (int i = 0; i < DN; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

  for (int j = 0; j < n_kv; ++j) {
    const int buf = j & 1;
    if (j + 1 < n_kv) {
      load_kv(j + 1, buf ^ 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (j == 0) {
#pragma unroll
      for (int kk = 0; kk < KS; ++kk) {
        const int mat = lane >> 3;
        const int r = warp * 16 + (lane & 7) + 8 * (mat & 1);
        const int c = kk * 16 + 8 * (mat >> 1);
        ldsm_x4(qf[kk], sQ + r * LDS + c);
      }
    }
    const __half* kb = sK + buf * BKV * LDS;
    const __half* vb = sV + buf * BKV * LDS;
    const bool pre = j < n_pre;
    const int key0 = (pre ? j : j - n_pre) * BKV;
    // 8-key column tiles this warp needs: all for prefix blocks, up to its last
    // query row on the causal diagonal; none when every row of the warp lies
    // past the sequence end (warp-uniform, so whole MMAs are skipped)
    int n_lim = 8;
    if (!pre) {
      const int last_row = min(wrow0 + 15, len - 1);
      n_lim = last_row < key0 ? 0 : min(8, (last_row - key0) / 8 + 1);
    }
    if (wrow0 >= len) n_lim = 0;

    if (n_lim > 0) {
      float sc[8][4];
#pragma unroll
      for (int n = 0; n < 8; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < KS; ++kk) {
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          if (2 * np < n_lim) {
            const int mat = lane >> 3;
            const int key = np * 16 + (lane & 7) + 8 * (mat >> 1);
            const int dim = kk * 16 + 8 * (mat & 1);
            uint32_t b[4];
            ldsm_x4(b, kb + key * LDS + dim);
            mma16816(sc[2 * np], qf[kk], b[0], b[1]);
            mma16816(sc[2 * np + 1], qf[kk], b[2], b[3]);
          }
        }
      }
      // scale into log2 units; mask prefix keys past P, future keys of the
      // sequence, keys past its end and the column tiles skipped above
      const bool need_mask = pre ? (key0 + BKV > P) : ((key0 + BKV - 1 > wrow0) || (key0 + BKV > len));
#pragma unroll
      for (int n = 0; n < 8; ++n) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          float v = sc[n][e] * scale_log2;
          if (need_mask) {
            const int key = key0 + n * 8 + 2 * tq + (e & 1);
            const int qr = wrow0 + gq + 8 * (e >> 1);
            if (pre ? key >= P : (key > qr || key >= len)) v = -INFINITY;
          }
          sc[n][e] = v;
        }
      }
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int n = 0; n < 8; ++n) {
        mx0 = fmaxf(mx0, fmaxf(sc[n][0], sc[n][1]));
        mx1 = fmaxf(mx1, fmaxf(sc[n][2], sc[n][3]));
      }
#pragma unroll
      for (int o2 = 1; o2 <= 2; o2 <<= 1) {
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o2));
      }
      const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
      const float base0 = mn0 == -INFINITY ? 0.f : mn0;
      const float base1 = mn1 == -INFINITY ? 0.f : mn1;
      const float c0 = exp2f(m0 - base0), c1 = exp2f(m1 - base1);
      m0 = mn0;
      m1 = mn1;
      float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
      for (int n = 0; n < 8; ++n) {
        sc[n][0] = exp2f(sc[n][0] - base0);
        sc[n][1] = exp2f(sc[n][1] - base0);
        sc[n][2] = exp2f(sc[n][2] - base1);
        sc[n][3] = exp2f(sc[n][3] - base1);
        rs0 += sc[n][0] + sc[n][1];
        rs1 += sc[n][2] + sc[n][3];
      }
      l0 = l0 * c0 + rs0;
      l1 = l1 * c1 + rs1;
#pragma unroll
      for (int i = 0; i < DN; ++i) {
        o[i][0] *= c0;
        o[i][1] *= c0;
        o[i][2] *= c1;
        o[i][3] *= c1;
      }
#pragma unroll
      for (int k2 = 0; k2 < 4; ++k2) {
        if (2 * k2 < n_lim) {
          uint32_t pa[4];
          pa[0] = pack_h2(sc[2 * k2][0], sc[2 * k2][1]);
          pa[1] = pack_h2(sc[2 * k2][2], sc[2 * k2][3]);
          pa[2] = pack_h2(sc[2 * k2 + 1][0], sc[2 * k2 + 1][1]);
          pa[3] = pack_h2(sc[2 * k2 + 1][2], sc[2 * k2 + 1][3]);
#pragma unroll
          for (int dp = 0; dp < DN / 2; ++dp) {
            const int mat = lane >> 3;
            const int key = k2 * 16 + (lane & 7) + 8 * (mat & 1);
            const int dim = dp * 16 + 8 * (mat >> 1);
            uint32_t b[4];
            ldsm_x4_t(b, vb + key * LDS + dim);
            mma16816(o[2 * dp], pa, b[0], b[1]);
            mma16816(o[2 * dp + 1], pa, b[2], b[3]);
          }
        }
      }
    }
    __syncthreads();
  }

#pragma unroll
  for (int o2 = 1; o2 <= 2; o2 <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, o2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, o2);
  }
  const float inv0 = l0 > 0.f ? 1.f / l0 : 0.f;
  const float inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
  const int64_t ldo = static_cast<int64_t>(Hq) * HD;
  const int r0 = wrow0 + gq, r1 = wrow0 + gq + 8;
#pragma unroll
  for (int i = 0; i < DN; ++i) {
    const int col = h * HD + i * 8 + 2 * tq;
    if (r0 < len)
      *reinterpret_cast<uint32_t*>(out + static_cast<int64_t>(st + r0) * ldo + col) = pack_h2(o[i][0] * inv0, o[i][1] * inv0);
    if (r1 < len)
      *reinterpret_cast<uint32_t*>(out + static_cast<int64_t>(st + r1) * ldo + col) = pack_h2(o[i][2] * inv1, o[i][3] * inv1);
  }
}

template <int HD>
void launch_hd(const __half* qkv, const int32_t* seq_start, const int32_t* tile_seq, const int32_t* tile_q0,
               int n_tiles_max, const int32_t* n_tiles_dev, int Hq, int Hkv, const __half* pkv, int P, __half* out,
               cudaStream_t s) {
  constexpr int LDS = HD + 8;
  const int smem = (BQ + 4 * BKV) * LDS * 2;
  cudaFuncSetAttribute(k_attention<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(HD));
  dim3 grid(n_tiles_max, Hq);
  k_attention<HD><<<grid, kThreads, smem, s>>>(qkv, seq_start, tile_seq, tile_q0, n_tiles_dev, Hq, Hkv, pkv, P,
                                               scale_log2, out);
}

}  // namespace

void launch_attention(const __half* qkv, int64_t /*T*/, const int32_t* seq_start, const int32_t* tile_seq,
                      const int32_t* tile_q0, int n_tiles_max, const int32_t* n_tiles_dev, int Hq, int Hkv, int hd,
                      const __half* prefix_kv, int P, __half* out, int* /*err*/, cudaStream_t s) {
  if (n_tiles_max <= 0) return;
  if (!prefix_kv) P = 0;
  switch (hd) {
    case 32: launch_hd<32>(qkv, seq_start, tile_seq, tile_q0, n_tiles_max, n_tiles_dev, Hq, Hkv, prefix_kv, P, out, s); break;
    case 64: launch_hd<64>(qkv, seq_start, tile_seq, tile_q0, n_tiles_max, n_tiles_dev, Hq, Hkv, prefix_kv, P, out, s); break;
    case 128: launch_hd<128>(qkv, seq_start, tile_seq, tile_q0, n_tiles_max, n_tiles_dev, Hq, Hkv, prefix_kv, P, out, s); break;
  }
}

}  // namespace aiq
