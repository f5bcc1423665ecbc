// Causal grouped-query attention on the 5th-generation tensor cores.
//
// One work item = (32 consecutive tokens of one sequence) x (the 4 query heads
// sharing one key/value head): its 128 query rows fill the M = 128 rows of a
// tcgen05 MMA, so every key/value block is fetched once per head group.  The
// keys of the shared prompt prefix (computed once per query, in prefix_kv)
// come first, then the sequence's own keys up to the tile's last token.
//
//   warp 0    TMA: the Q tile (3-D box hd x heads x tokens) into one of two
//             slots, then K and V blocks of 64 keys into two separate rings of
//             NKV slots (128-byte swizzle).  A K slot is free once the S MMA
//             that read it has completed, a V slot once the PV MMA that read
//             it has, so a block's loads are issued NKV blocks ahead.  The
//             same thread publishes each item's bounds (sequence start and
//             length, first token, key/value head) in a four-slot shared
//             ring, so the softmax warps never wait on global loads between
//             items.
//   warp 1    tcgen05.mma: S = Q K^T into one of two 64-column TMEM score
//             buffers, and O += P V into the item's TMEM output accumulator,
//             with P read from TMEM (it overwrites its own scores) and V read
//             as an MN-major operand straight from its TMA tile.
//   warps 2-5 one query row per thread: read its 64 scores with tcgen05.ld,
//             apply the causal / prefix / length mask, keep the running max
//             (the output is rescaled only when the max grows by more than
//             2^8, so P never exceeds 256), and write exp2(s - max) as fp16
//             pairs back over the first 32 columns of the same score buffer
//             with tcgen05.st; an item's output is divided by the row sum and
//             stored after the next item's first block: through a shared
//             staging tile and one TMA store when all the tile's tokens
//             belong to its sequence, row by row otherwise.
//
// Ordering without extra waits: the MMA warp issues S(g+1) before PV(g), and
// tcgen05 MMAs of one thread run in issue order, so S(g+2), which reuses the
// score buffer of block g, only starts after PV(g) has read P(g).  The commit
// that signals S(g) tracks every earlier MMA of the thread, so a softmax
// thread that has seen S(g) complete knows PV(g-2) has too: its parity waits
// on the two PV barriers can never be a full phase behind.  The softmax warps
// signal P on one barrier per score buffer: S(g+1) is ready before PV(g) is
// issued, so one warp may finish block g+1 while another still writes P(g),
// and on a single barrier its second arrival would complete block g's phase
// early; a warp cannot reach block g+2 before PV(g), so two barriers suffice.
// Work items are persistent per CTA; every wait is bounded.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"

namespace aiq {
namespace {

constexpr int kThreadsTC = 192;
constexpr int kKeys = 64;  // keys per block

template <int HD>
struct ACfg {
  static constexpr int NC = HD / 64;             // 64-column sub-tiles of one head
  static constexpr int NKV = 3;                  // slots of the K ring and of the V ring
  static constexpr int Q_BYTES = 128 * HD * 2;   // 128 rows
  static constexpr int SUB = 64 * 128;           // one [64 x 64] fp16 sub-tile
  static constexpr int K_BYTES = NC * SUB;
  static constexpr int OFF_Q = 0;                // two slots
  static constexpr int OFF_K = OFF_Q + 2 * Q_BYTES;
  static constexpr int OFF_V = OFF_K + NKV * K_BYTES;
  static constexpr int OFF_OUT = OFF_V + NKV * K_BYTES;  // output staging tile (TMA store source)
  static constexpr int OFF_INFO = OFF_OUT + Q_BYTES;     // item bounds ring, 4 x int4
  static constexpr int OFF_BAR = OFF_INFO + 4 * 16;
  static constexpr int N_BARS = 4 + 4 * NKV + 2 + 2 + 2 + 2 + 1 + 4 + 4 + 2;
  static constexpr int SMEM = 1024 + OFF_BAR + N_BARS * 8 + 16;
  // two 64-column score buffers, then two HD-column output accumulators (one
  // per alternating work item), rounded up to a power of two
  static constexpr int TMEM_COLS = HD == 64 ? 256 : 512;
  static constexpr int O_COL = 128;
};
// two CTAs per SM at HD = 64 (each also keeps 1 KB of the SM's shared memory)
static_assert(2 * (ACfg<64>::SMEM + 1024) <= 233472, "HD = 64 tiles must fit two CTAs per SM");
static_assert(ACfg<128>::SMEM <= 232448, "HD = 128 tiles must fit one CTA");

struct AttnArgs {
  const int32_t* seq_start;
  const int32_t* tile_seq;
  const int32_t* tile_q0;
  const int32_t* n_tiles;
  int Hq, Hkv, G, TQ, P;
  float scale_log2;
  __half* out;
  int* err;
};

__device__ __forceinline__ void load2x32_f(uint32_t ta, uint32_t tb, float* va, float* vb) {
  uint32_t ra[32], rb[32];
  tmem_ld_32x32b_x32(ta, ra);
  tmem_ld_32x32b_x32(tb, rb);
  tmem_ld_wait();
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    va[j] = __uint_as_float(ra[j]);
    vb[j] = __uint_as_float(rb[j]);
  }
}

// 2^x with the SFU's approximation (relative error ~2^-22, flushes
// subnormals): plenty for probabilities that are rounded to fp16 next.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Packed fp32 pairs (Blackwell f32x2): two IEEE fma / add per instruction,
// each lane's result identical to the scalar operation.
__device__ __forceinline__ unsigned long long f2_bits(float2 v) {
  return (static_cast<unsigned long long>(__float_as_uint(v.y)) << 32) | __float_as_uint(v.x);
}
__device__ __forceinline__ float2 bits_f2(unsigned long long b) {
  return make_float2(__uint_as_float(static_cast<uint32_t>(b)), __uint_as_float(static_cast<uint32_t>(b >> 32)));
}
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  unsigned long long r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(f2_bits(a)), "l"(f2_bits(b)), "l"(f2_bits(c)));
  return bits_f2(r);
}
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
  unsigned long long r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(f2_bits(a)), "l"(f2_bits(b)));
  return bits_f2(r);
}

// Shared -> global tile copy by the TMA unit (3-D box), in a bulk async-group.
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, const void* smem_src, int x, int y, int z) {
  asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.tile.bulk_group [%0, {%1, %2, %3}], [%4];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(z), "r"(smem_u32(smem_src))
               : "memory");
}

// MN-major operand (N contiguous) in the 128-byte swizzle: rows of 64 N
// elements, 8-row groups 1024 B apart along K, 64-column atoms 8 KB apart along N.
__device__ __forceinline__ uint64_t smem_desc_mn_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(lbo >> 4) << 16;
  d |= static_cast<uint64_t>(sbo >> 4) << 32;
  d |= static_cast<uint64_t>(1u) << 46;
  d |= static_cast<uint64_t>(2u) << 61;
  return d;
}

// D (TMEM) (+)= A (TMEM: lane = row, two fp16 per 32-bit column along K) * B (smem).
__device__ __forceinline__ void umma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

template <int HD>
__global__ void __launch_bounds__(kThreadsTC, HD == 64 ? 2 : 1)
    k_attention_tc(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kv,
                   const __grid_constant__ CUtensorMap tm_pre, const __grid_constant__ CUtensorMap tm_out, AttnArgs a) {
  using C = ACfg<HD>;
  constexpr int NKV = C::NKV;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* q_full = bars + 0;             // [2]
  uint64_t* q_empty = bars + 2;            // [2]: the item's S MMAs have completed
  uint64_t* k_full = bars + 4;             // [NKV]
  uint64_t* k_empty = k_full + NKV;        // [NKV]: the S MMA of the block has completed
  uint64_t* v_full = k_empty + NKV;        // [NKV]
  uint64_t* v_empty = v_full + NKV;        // [NKV]: the PV MMA of the block has completed
  uint64_t* s_full = v_empty + NKV;        // [2]
  uint64_t* p_full = s_full + 2;           // [2]: P of block g written over its scores (score buffer g & 1)
  uint64_t* o_done = p_full + 2;           // [2]: PV of block g commits o_done[g & 1]
  uint64_t* o_free = o_done + 2;           // [2]: output accumulator it & 1 read out
  uint64_t* mma_done = o_free + 2;
  uint64_t* info_full = mma_done + 1;      // [4]: item bounds published by the TMA thread
  uint64_t* info_empty = info_full + 4;    // [4]: read by the four softmax warps
  uint64_t* out_full = info_empty + 4;     // the staging tile holds an item's output (4 warps)
  uint64_t* out_free = out_full + 1;       // the previous TMA store has read the staging tile
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(out_free + 1);
  int4* info = reinterpret_cast<int4*>(smem + C::OFF_INFO);
  uint8_t* sOut = smem + C::OFF_OUT;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  auto sQ = [&](int b) { return smem + C::OFF_Q + b * C::Q_BYTES; };
  auto sK = [&](int b) { return smem + C::OFF_K + b * C::K_BYTES; };
  auto sV = [&](int b) { return smem + C::OFF_V + b * C::K_BYTES; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int* err = a.err;
  if (threadIdx.x == 0) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(&q_full[b], 1);
      mbar_init(&q_empty[b], 1);
      mbar_init(&s_full[b], 1);
      mbar_init(&p_full[b], 4);
      mbar_init(&o_done[b], 1);
      mbar_init(&o_free[b], 4);
    }
    for (int b = 0; b < NKV; ++b) {
      mbar_init(&k_full[b], 1);
      mbar_init(&k_empty[b], 1);
      mbar_init(&v_full[b], 1);
      mbar_init(&v_empty[b], 1);
    }
    mbar_init(mma_done, 1);
    for (int b = 0; b < 4; ++b) {
      mbar_init(&info_full[b], 1);
      mbar_init(&info_empty[b], 4);
    }
    mbar_init(out_full, 4);
    mbar_init(out_free, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_kv);
    tma_prefetch_desc(&tm_pre);
    tma_prefetch_desc(&tm_out);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int n_work = *a.n_tiles * a.Hkv;
  const int n_pre = (a.P + kKeys - 1) / kKeys;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA
      uint32_t g = 0;   // key blocks whose K load was issued (ring position)
      uint32_t gv = 0;  // key blocks whose V load was issued
      int it = 0;       // Q loads issued
      bool ok = true;
      for (int w = blockIdx.x; w < n_work && ok; w += gridDim.x) {
        const int tidx = w / a.Hkv, kvh = w % a.Hkv;
        const int s = a.tile_seq[tidx], q0 = a.tile_q0[tidx];
        const int st = a.seq_start[s], len = a.seq_start[s + 1] - st;
        const int q_end = min(q0 + a.TQ, len);
        const int n_kv = n_pre + (q_end + kKeys - 1) / kKeys;
        // the softmax warps take the item's bounds from this ring instead of
        // reading them from global memory at every item start
        const int is = it & 3;
        if (!mbar_wait_bounded(&info_empty[is], ((it >> 2) & 1) ^ 1, abort_flag, err)) break;
        info[is] = make_int4(st, len, q0, kvh);
        mbar_arrive(&info_full[is]);
        const int qb = it & 1;
        if (!mbar_wait_bounded(&q_empty[qb], ((it >> 1) & 1) ^ 1, abort_flag, err)) break;
        mbar_arrive_expect_tx(&q_full[qb], C::Q_BYTES);
        ++it;
        for (int c = 0; c < C::NC; ++c)
          tma_load_3d(sQ(qb) + c * (128 * 128), &tm_q, &q_full[qb], c * 64, kvh * a.G, st + q0);
        for (int j = 0; j < n_kv; ++j, ++g) {
          const int b = g % NKV;
          const uint32_t ph = ((g / NKV) & 1) ^ 1;
          const bool pre = j < n_pre;
          const CUtensorMap* map = pre ? &tm_pre : &tm_kv;
          const int kcol = pre ? kvh * HD : (a.Hq + kvh) * HD;
          const int vcol = pre ? (a.Hkv + kvh) * HD : (a.Hq + a.Hkv + kvh) * HD;
          const int row = pre ? j * kKeys : st + (j - n_pre) * kKeys;
          if (!mbar_wait_bounded(&k_empty[b], ph, abort_flag, err)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&k_full[b], C::K_BYTES);
          for (int c = 0; c < C::NC; ++c) tma_load_2d(sK(b) + c * C::SUB, map, &k_full[b], kcol + c * 64, row);
          if (!mbar_wait_bounded(&v_empty[b], ph, abort_flag, err)) {
            ok = false;
            ++g;  // this block's K load is in flight, its V load is not
            break;
          }
          mbar_arrive_expect_tx(&v_full[b], C::K_BYTES);
          for (int c = 0; c < C::NC; ++c) tma_load_2d(sV(b) + c * C::SUB, map, &v_full[b], vcol + c * 64, row);
          ++gv;
        }
      }
      if (!ok || *abort_flag) {
        // let this thread's copies still in flight land before the CTA can exit
        // (the last use of each slot is the only one that can be outstanding)
        volatile int never = 0;
        for (uint32_t i = g > NKV ? g - NKV : 0; i < g; ++i)
          mbar_wait_bounded(&k_full[i % NKV], (i / NKV) & 1, &never, nullptr, 200000000ull);
        for (uint32_t i = gv > NKV ? gv - NKV : 0; i < gv; ++i)
          mbar_wait_bounded(&v_full[i % NKV], (i / NKV) & 1, &never, nullptr, 200000000ull);
        for (int i = it > 2 ? it - 2 : 0; i < it; ++i)
          mbar_wait_bounded(&q_full[i & 1], (i >> 1) & 1, &never, nullptr, 200000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA
      constexpr uint32_t idesc_s = idesc_f16_f32(128, kKeys);
      constexpr uint32_t idesc_o = idesc_f16_f32(128, HD) | (1u << 16);  // B (= V) MN-major
      uint32_t g = 0;
      int it = 0;
      bool ok = true;
      auto issue_s = [&](uint32_t gg, int qb) -> bool {
        const int kb = gg % NKV;
        if (!mbar_wait_bounded(&k_full[kb], (gg / NKV) & 1, abort_flag, err)) return false;
        tc_fence_after();
        const uint32_t d = tmem_base + (gg & 1) * kKeys;
#pragma unroll
        for (int c = 0; c < C::NC; ++c)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            umma_f16_ss(d, smem_desc_k_sw128(smem_u32(sQ(qb) + c * (128 * 128)) + k * 32),
                        smem_desc_k_sw128(smem_u32(sK(kb) + c * C::SUB) + k * 32), idesc_s, (c | k) != 0);
        umma_commit(&k_empty[kb]);
        umma_commit(&s_full[gg & 1]);
        return true;
      };
      // key blocks of an item (the shared prefix's, then the row's own up to
      // the tile's last token)
      auto blocks_of = [&](int w) -> int {
        const int tidx = w / a.Hkv;
        const int s = a.tile_seq[tidx], q0 = a.tile_q0[tidx];
        const int len = a.seq_start[s + 1] - a.seq_start[s];
        return n_pre + (min(q0 + a.TQ, len) + kKeys - 1) / kKeys;
      };
      // The blocks of all this CTA's items form one stream: the scores of the
      // next block, also the first block of the next item, are issued before
      // this block's PV, so an item boundary costs no extra hand-off.
      int w = blockIdx.x;
      if (w < n_work) {
        int n_kv = blocks_of(w);
        if (!mbar_wait_bounded(&q_full[0], 0, abort_flag, err) || (tc_fence_after(), !issue_s(g, 0))) ok = false;
        while (ok) {
          const int qb = it & 1;
          const int w_next = w + gridDim.x;
          const int n_next = w_next < n_work ? blocks_of(w_next) : 0;
          for (int j = 0; j < n_kv; ++j, ++g) {
            if (j + 1 < n_kv) {
              if (!issue_s(g + 1, qb)) {
                ok = false;
                break;
              }
            } else {
              umma_commit(&q_empty[qb]);  // all S MMAs of this item issued
              if (n_next > 0) {
                const int it1 = it + 1;
                if (!mbar_wait_bounded(&q_full[it1 & 1], (it1 >> 1) & 1, abort_flag, err)) {
                  ok = false;
                  break;
                }
                tc_fence_after();
                if (!issue_s(g + 1, it1 & 1)) {
                  ok = false;
                  break;
                }
              }
            }
            if (!mbar_wait_bounded(&p_full[g & 1], (g >> 1) & 1, abort_flag, err)) {
              ok = false;
              break;
            }
            // the first PV overwrites this item's accumulator: the softmax warps
            // must have read out the output of the item two back
            if (j == 0 && !mbar_wait_bounded(&o_free[qb], ((it >> 1) & 1) ^ 1, abort_flag, err)) {
              ok = false;
              break;
            }
            const int vb = g % NKV;
            if (!mbar_wait_bounded(&v_full[vb], (g / NKV) & 1, abort_flag, err)) {
              ok = false;
              break;
            }
            tc_fence_after();
#pragma unroll
            for (int k = 0; k < 4; ++k)
              umma_f16_ts(tmem_base + C::O_COL + qb * HD, tmem_base + (g & 1) * kKeys + k * 8,
                          smem_desc_mn_sw128(smem_u32(sV(vb)) + k * 2048, HD == 64 ? 1024u : 8192u, 1024u),
                          idesc_o, (j | k) != 0);
            umma_commit(&v_empty[vb]);
            umma_commit(&o_done[g & 1]);
          }
          if (!ok || n_next == 0) break;
          w = w_next;
          n_kv = n_next;
          ++it;
        }
      }
      umma_commit(mma_done);
      volatile int never = 0;
      mbar_wait_bounded(mma_done, 0, &never, err);
    }
  } else {
    // ------------------------------------------------- softmax / epilogue
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;  // TMEM lane = query row of the tile
    const int t = r / a.G, gq = r % a.G;
    const uint32_t trow = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16);
    uint32_t g = 0;
    int it = 0;
    bool ok = true;
    // PV of block gg done (o_done completes once per block on slot gg & 1;
    // this thread has already seen PV of block gg - 2 complete, and PV of
    // block gg + 2 needs a P that it has not yet written, so parity is exact)
    // Every wait of these warps is taken warp-uniformly: a lane that gives up
    // (timeout or abort) makes the whole warp give up, so no lane is left
    // alone in the warp-synchronous tcgen05 loads and stores that follow.
    auto wait_all = [&](uint64_t* bar, uint32_t parity) -> bool {
      return __all_sync(0xffffffffu, mbar_wait_bounded(bar, parity, abort_flag, err));
    };
    auto wait_pv = [&](uint32_t gg) -> bool { return wait_all(&o_done[gg & 1], (gg >> 1) & 1); };
    // The output of an item is read out after the next item's first block
    // (its last PV may still be running meanwhile): O / l, stored for the
    // tile's real tokens, then the accumulator is handed back to the MMA warp.
    // A tile whose tokens all belong to its sequence is written by one TMA
    // store of the CTA's staging tile (rows in TMEM-lane order = the box's
    // token-major, head-minor order, 128-byte swizzle); a ragged last tile is
    // written row by row, live rows only, since its box would reach into the
    // next sequence's tokens.  nf counts the full-tile read-outs: the k-th
    // waits for out_free phase k - 1 (the store of read-out k - 1 has read
    // the staging tile) and its four warps complete out_full phase k.
    struct Pending {
      bool on, live, full;
      int buf, kvh, tok;
      uint32_t g_last;
      float inv;
      __half* dst;
    } pend{false, false, false, 0, 0, 0, 0, 0.f, nullptr};
    uint32_t nf = 0;
    const bool issuer = threadIdx.x == 64;
    auto flush = [&]() -> bool {
      if (!wait_pv(pend.g_last)) return false;
      tc_fence_after();
      if (pend.full) {
        if (nf > 0) {
          if (issuer) {
            bulk_wait_group_read<0>();
            mbar_arrive(out_free);
          }
          if (!wait_all(out_free, (nf - 1) & 1)) return false;
        }
      }
      const uint32_t ocol = trow + C::O_COL + pend.buf * HD;
#pragma unroll 1
      for (int c = 0; c < HD; c += 32) {
        uint32_t o[32];
        tmem_ld_32x32b_x32(ocol + c, o);
        tmem_ld_wait();
        if (pend.full) {
          uint8_t* row = sOut + (c >> 6) * (128 * 128) + r * 128;
#pragma unroll
          for (int q4 = 0; q4 < 4; ++q4) {
            uint32_t pk[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              __half2 h = __floats2half2_rn(__uint_as_float(o[q4 * 8 + 2 * i]) * pend.inv,
                                            __uint_as_float(o[q4 * 8 + 2 * i + 1]) * pend.inv);
              pk[i] = *reinterpret_cast<uint32_t*>(&h);
            }
            const int chunk = ((c & 63) >> 3) + q4;
            *reinterpret_cast<uint4*>(row + ((chunk ^ (r & 7)) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
          }
        } else if (pend.live) {
          uint4* d4 = reinterpret_cast<uint4*>(pend.dst + c);
#pragma unroll
          for (int q4 = 0; q4 < 4; ++q4) {
            uint32_t pk[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              __half2 h = __floats2half2_rn(__uint_as_float(o[q4 * 8 + 2 * i]) * pend.inv,
                                            __uint_as_float(o[q4 * 8 + 2 * i + 1]) * pend.inv);
              pk[i] = *reinterpret_cast<uint32_t*>(&h);
            }
            d4[q4] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
          }
        }
      }
      tc_fence_before();
      if (pend.full) fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&o_free[pend.buf]);
        if (pend.full) mbar_arrive(out_full);
      }
      if (pend.full) {
        // the storing thread's wait decides for its whole warp
        bool stored = true;
        if (issuer) {
          stored = mbar_wait_bounded(out_full, nf & 1, abort_flag, err);
          if (stored) {
#pragma unroll
            for (int cc = 0; cc < C::NC; ++cc)
              tma_store_3d(&tm_out, sOut + cc * (128 * 128), cc * 64, pend.kvh * a.G, pend.tok);
            bulk_commit_group();
          }
        }
        if (!__shfl_sync(0xffffffffu, stored, 0)) return false;
        ++nf;
      }
      pend.on = false;
      return true;
    };
    for (int w = blockIdx.x; w < n_work && ok; w += gridDim.x, ++it) {
      const int is = it & 3;
      if (!wait_all(&info_full[is], (it >> 2) & 1)) {
        ok = false;
        break;
      }
      const int4 inf = info[is];
      __syncwarp();
      if (lane == 0) mbar_arrive(&info_empty[is]);
      const int st = inf.x, len = inf.y, q0 = inf.z, kvh = inf.w;
      const int q_end = min(q0 + a.TQ, len);
      const int n_kv = n_pre + (q_end + kKeys - 1) / kKeys;
      const int qpos = q0 + t;
      const uint32_t ocol = trow + C::O_COL + (it & 1) * HD;
      float m_used = 0.f, l = 0.f;
      for (int j = 0; j < n_kv; ++j, ++g) {
        const int b = g & 1;
        if (!wait_all(&s_full[b], (g >> 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        float v[64];
        load2x32_f(trow + b * kKeys, trow + b * kKeys + 32, v, v + 32);
        const bool pre = j < n_pre;
        const int key0 = (pre ? j : j - n_pre) * kKeys;
        // warp-uniform: only the prefix's last block and the causal diagonal /
        // sequence end need a mask; then key c is visible iff c < lim
        const bool need_mask = pre ? (key0 + kKeys > a.P) : (key0 + kKeys - 1 > q0 || key0 + kKeys > len);
        if (need_mask) {
          const int lim = pre ? a.P - key0 : min(qpos + 1, len) - key0;
#pragma unroll
          for (int c = 0; c < 64; ++c) v[c] = c < lim ? v[c] : -INFINITY;
        }
        // running max on the raw scores; the softmax scale (with log2 e) is
        // folded into one FFMA inside the exponent below
        // (eight independent partial maxima keep the FMNMX chain short)
        float pm[8];
#pragma unroll
        for (int c = 0; c < 8; ++c) pm[c] = v[c];
#pragma unroll
        for (int c = 8; c < 64; ++c) pm[c & 7] = fmaxf(pm[c & 7], v[c]);
        const float mr = fmaxf(fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3])),
                               fmaxf(fmaxf(pm[4], pm[5]), fmaxf(pm[6], pm[7])));
        const float mx = mr * a.scale_log2;
        if (j == 0) {
          m_used = mx == -INFINITY ? 0.f : mx;
        } else {
          const bool grow = mx > m_used + 8.f;
          if (__any_sync(0xffffffffu, grow)) {
            // rescale this warp's output rows once the previous block's PV is done
            if (!wait_pv(g - 1)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const float f = grow ? ex2_approx(m_used - mx) : 1.f;
            if (grow) {
              l *= f;
              m_used = mx;
            }
#pragma unroll 1
            for (int c = 0; c < HD; c += 32) {
              uint32_t o[32];
              tmem_ld_32x32b_x32(ocol + c, o);
              tmem_ld_wait();
#pragma unroll
              for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * f);
              tmem_st_32x32b_x32(ocol + c, o);
            }
            tmem_st_wait();
          }
        }
        float2 ps[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
        const float2 sc2 = make_float2(a.scale_log2, a.scale_log2), nm2 = make_float2(-m_used, -m_used);
        uint32_t pk[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float2 x = ffma2(make_float2(v[2 * i], v[2 * i + 1]), sc2, nm2);
          const float2 p = make_float2(ex2_approx(x.x), ex2_approx(x.y));
          ps[i & 3] = fadd2(ps[i & 3], p);
          __half2 h = __floats2half2_rn(p.x, p.y);
          pk[i] = *reinterpret_cast<uint32_t*>(&h);
        }
        l += ((ps[0].x + ps[0].y) + (ps[1].x + ps[1].y)) + ((ps[2].x + ps[2].y) + (ps[3].x + ps[3].y));
        // P (fp16 pairs) over the first 32 columns of this block's score buffer
        tmem_st_32x32b_x32(trow + b * kKeys, pk);
        tmem_st_wait();
        tc_fence_before();  // this block's score reads and P writes are complete
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[b]);
        if (j == 0 && pend.on && !flush()) {
          ok = false;
          break;
        }
      }
      if (!ok) break;
      pend.on = true;
      pend.live = qpos < len;
      pend.full = q0 + a.TQ <= len;
      pend.kvh = kvh;
      pend.tok = st + q0;
      pend.buf = it & 1;
      pend.g_last = g - 1;
      pend.inv = l > 0.f ? 1.f / l : 0.f;
      pend.dst = a.out + static_cast<int64_t>(st + qpos) * (a.Hq * HD) + (kvh * a.G + gq) * HD;
    }
    if (ok && pend.on) flush();
    // the CTA's shared memory must outlive the TMA stores that read it
    if (issuer) bulk_wait_group_all();
  }

  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn_attn() {
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

bool map2d(CUtensorMap* m, const __half* base, int64_t rows, int64_t cols) {
  auto fn = encode_fn_attn();
  if (!fn) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols * 2)};
  cuuint32_t box[2] = {64, 64};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<__half*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// qkv viewed as [T][heads][hd]; box = 64 columns x G heads x TQ tokens.
bool map3d_q(CUtensorMap* m, const __half* base, int64_t T, int heads, int hd, int G, int TQ) {
  auto fn = encode_fn_attn();
  if (!fn) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(hd), static_cast<cuuint64_t>(heads), static_cast<cuuint64_t>(T)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(hd * 2), static_cast<cuuint64_t>(int64_t(heads) * hd * 2)};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(G), static_cast<cuuint32_t>(TQ)};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<__half*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int HD>
int launch_tc(const CUtensorMap& mq, const CUtensorMap& mkv, const CUtensorMap& mpre, const CUtensorMap& mout,
              const AttnArgs& a,
              int n_work_max, int num_sms, cudaStream_t s) {
  using C = ACfg<HD>;
  cudaError_t e = cudaFuncSetAttribute(k_attention_tc<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  const int per_sm = C::SMEM <= 113 * 1024 ? 2 : 1;
  const int grid = n_work_max < num_sms * per_sm ? n_work_max : num_sms * per_sm;
  if (grid <= 0) return 0;
  k_attention_tc<HD><<<grid, kThreadsTC, C::SMEM, s>>>(mq, mkv, mpre, mout, a);
  return cudaGetLastError();
}

}  // namespace

bool attention_tc_supported(int hd, int Hq, int Hkv) {
  if (hd != 64 && hd != 128) return false;
  const int G = Hq / Hkv;
  return Hq % Hkv == 0 && G >= 1 && G <= 128 && 128 % G == 0;
}

int attention_tc_tile_tokens(int Hq, int Hkv) { return 128 / (Hq / Hkv); }

int launch_attention_tc(const __half* qkv, int64_t T, const int32_t* seq_start, const int32_t* tile_seq,
                        const int32_t* tile_q0, int n_tiles_max, const int32_t* n_tiles_dev, int Hq, int Hkv, int hd,
                        const __half* prefix_kv, int P, __half* out, int* err, int num_sms, cudaStream_t s) {
  if (n_tiles_max <= 0 || T <= 0) return 0;
  const int G = Hq / Hkv, TQ = 128 / G;
  const int heads = Hq + 2 * Hkv;
  CUtensorMap mq, mkv, mpre, mout;
  if (!map3d_q(&mq, qkv, T, heads, hd, G, TQ) || !map2d(&mkv, qkv, T, int64_t(heads) * hd) ||
      !map3d_q(&mout, out, T, Hq, hd, G, TQ))
    return cudaErrorInvalidValue;
  if (prefix_kv && P > 0) {
    if (!map2d(&mpre, prefix_kv, P, int64_t(2) * Hkv * hd)) return cudaErrorInvalidValue;
  } else {
    mpre = mkv;
    P = 0;
  }
  AttnArgs a{seq_start, tile_seq, tile_q0, n_tiles_dev, Hq, Hkv, G, TQ, P,
             1.4426950408889634f / sqrtf(static_cast<float>(hd)), out, err};
  const int n_work_max = n_tiles_max * Hkv;
  return hd == 64 ? launch_tc<64>(mq, mkv, mpre, mout, a, n_work_max, num_sms, s)
                  : launch_tc<128>(mq, mkv, mpre, mout, a, n_work_max, num_sms, s);
}

}  // namespace aiq
