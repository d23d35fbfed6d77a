// Chunk-window flash attention on tcgen05 (Sec. 3.3 "Attention Pattern", Eq. kv_cache).
//
// Keys are the first n_keys rows of the layer's ring: ring slots 0..c-1 always hold exactly
// the c = min(t+1, W) cached chunks, keys carry their RoPE rotation from the append, and
// softmax does not depend on key order, so no mask tensor is needed; only the ragged last key
// block is cut at n_keys. GQA: head n reads KV group n / (N / G).
//
// GQA row packing: the query rows of the heads sharing KV group g form one row space (head
// after head, each head's Lq rows padded to lq_pad, a multiple of 8). One CTA = two consecutive
// 128-row tiles X = 0, 1 of one group's row space, so each K / V block is loaded once for both
// and the only padding is at the end of the group, not at the end of every head.
// Optionally the key range is split over `splits` CTAs whose partial results a second kernel
// combines (balances the grid over the SMs).
//
// TMEM (512 columns): per tile X, S_X (128 fp32 columns), P_X (64 columns, 128 keys of fp16
// packed in pairs) and O_X (64 fp32 columns). S and P are separate, so the MMA for the next
// key block's S can run as soon as the softmax has read the current S, while P is still being
// computed: each tile's softmax warps go from block to block without waiting on the tensor
// core, and the two tiles' MMAs interleave on it.
//   S_X(j)  = Q_X K_j^T     tcgen05.mma M=128 N=128 K=64 (A, B from shared memory)
//   O_X    += P_X(j) V_j    M=128 N=64 K=128, fp16 x fp16: A = P_X read from TMEM, B = V^T
//                           from the transposed fp16 V ring
// Warp roles (352 threads):
//   warp 8        TMA: Q tiles once, then K and V^T blocks of 128 keys into a 3-stage ring
//   warps 9 / 10  one thread each issues tile 0's / tile 1's MMAs: S of block j+1 once the
//                 tile's softmax has read S(j), then P V of block j once P(j) is written
//   warps 0-3 / 4-7  softmax of tile 0 / 1, one query row (TMEM lane) per thread: load S,
//                 release it, running max in the log2 domain and running row sum in
//                 registers, P = exp2(s - m) as fp16 in registers, then into P_X once the
//                 previous P V has read it. The two tiles' warps on one SMSP alternate on the
//                 exponentials. O_X is rescaled in TMEM (load, multiply, store) only when a row's max
//                 grows by more than 2^8, so P stays <= 256 and the rescale is rare.
#include "fd_internal.h"
#include "fd_ptx.cuh"

namespace fd {

namespace attn {
constexpr int kStages = 3;
constexpr int kQBytes = 128 * 128;           // Q tile [128 rows][64] bf16
constexpr int kKBytes = 128 * 128;           // K block [128 keys][64] bf16
constexpr int kVSub = 64 * 128;              // V^T sub-tile [64 dims][64 keys] bf16
constexpr int kVBytes = 2 * kVSub;           // V^T block of 128 keys
constexpr int kOffQ = 0;
constexpr int kOffK = 2 * kQBytes;
constexpr int kOffV = kOffK + kStages * kKBytes;
constexpr int kOffBar = kOffV + kStages * kVBytes;
constexpr int kSmem = kOffBar + 256;
constexpr int kThreads = 352;
constexpr int kTmemCols = 512;
constexpr uint32_t kColS = 0, kColP = 256, kColO = 384;  // + 128 X, + 64 X, + 64 X
constexpr float kRescaleLog2 = 8.0f;
// barrier indices
constexpr int kBarQ = 0, kBarKvFull = 1, kBarKvEmpty = kBarKvFull + kStages,
              kBarS = kBarKvEmpty + kStages,   // [tile] S_X(j) computed
              kBarSFree = kBarS + 2,           // [tile] S_X(j) read by the softmax
              kBarP = kBarSFree + 2,           // [tile] P_X(j) written
              kBarPv = kBarP + 2,              // [tile] P V of block j completed
              kBarDone = kBarPv + 2,           // [tile] every MMA of the tile's issuer completed
              kBarTurn = kBarDone + 2,  // [tile][quarter] the other tile's warp of this SMSP
                                        // has finished its exponentials: this tile's turn
              kNumBars = kBarTurn + 8;
static_assert(kNumBars * 8 + 4 <= 256, "barrier area");
static_assert(kSmem <= 227 * 1024, "shared memory");
}  // namespace attn

__device__ __forceinline__ float add_pair(uint32_t a, uint32_t b) {
  return __uint_as_float(a) + __uint_as_float(b);
}

__global__ void __launch_bounds__(attn::kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmQ8,
                const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const __grid_constant__ AttnParams p) {
  using namespace attn;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t base = smem_u32(smem);
  const bool aligned = (base & 1023u) == 0;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  const uint32_t bar0 = smem_u32(bars);
  auto bar = [&](int i) { return bar0 + 8u * static_cast<uint32_t>(i); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + kNumBars);

  // the two tiles of this CTA: packed rows (2 blockIdx.x + X) * 128 + i of KV group g
  const int g = blockIdx.y;
  const int hpg = p.heads / p.groups;

  if (threadIdx.x == 0) {
    if (!aligned) atomicOr(p.err, ERR_SMEM_ALIGN);
    mbar_init(bar(kBarQ), 1);
    for (int st = 0; st < kStages; ++st) {
      mbar_init(bar(kBarKvFull + st), 1);
      mbar_init(bar(kBarKvEmpty + st), 2);  // both tiles' issuers release a stage
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(bar(kBarS + x), 1);
      mbar_init(bar(kBarSFree + x), 128);
      mbar_init(bar(kBarP + x), 128);
      mbar_init(bar(kBarPv + x), 1);
      mbar_init(bar(kBarDone + x), 1);
    }
    for (int i = 0; i < 8; ++i) mbar_init(bar(kBarTurn + i), 1);
    fence_barrier_init();
  }
  grid_dep_wait();  // Q and the ring written by the previous kernels; TMEM freed by their CTAs
  int n_keys = p.n_keys_host;
  if (p.step_dev != nullptr) {
    const int t = *p.step_dev;
    n_keys = (t + 1 < p.window ? t + 1 : p.window) * p.rows_per_chunk;
  }
  const int nblk_all = (n_keys + 127) / 128;
  const int per = (nblk_all + p.splits - 1) / p.splits;
  const int kb0 = blockIdx.z * per;
  const int kb_end = kb0 + per < nblk_all ? kb0 + per : nblk_all;
  const int nblk = kb_end > kb0 ? kb_end - kb0 : 0;
  if (warp == 0) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 8) {
    // ------------------------------------------------------------ TMA loads
    if (lane == 0 && aligned && nblk > 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmQ8);
      prefetch_tmap(&tmK);
      prefetch_tmap(&tmV);
      mbar_expect_tx(bar(kBarQ), 2 * kQBytes);
      // A tile inside one head's rows is one 128-row box (rows past Lq read the fill value);
      // a tile across two heads is loaded in boxes of 8 rows (one 1024-byte swizzle atom
      // each, same shared-memory layout). Rows past the group's last head load head 0's
      // first rows; their outputs are not written.
      for (int x = 0; x < 2; ++x) {
        const int rho0 = (2 * blockIdx.x + x) * kBM;
        const int hl0 = rho0 / p.lq_pad;
        const int hl1 = (rho0 + kBM - 1) / p.lq_pad;
        const uint32_t dst = base + kOffQ + x * kQBytes;
        if (hl0 >= hpg) {
          tma_load_2d(dst, &tmQ, bar(kBarQ), g * hpg * kHeadDim, 0);
        } else if (hl1 == hl0 || hl1 >= hpg) {
          tma_load_2d(dst, &tmQ, bar(kBarQ), (g * hpg + hl0) * kHeadDim, rho0 - hl0 * p.lq_pad);
        } else {
          for (int b = 0; b < kBM / 8; ++b) {
            const int rho = rho0 + 8 * b;
            int hl = rho / p.lq_pad;
            int r = rho - hl * p.lq_pad;
            if (hl >= hpg) hl = r = 0;
            tma_load_2d(dst + b * 1024, &tmQ8, bar(kBarQ), (g * hpg + hl) * kHeadDim, r);
          }
        }
      }
      int j = 0;
      for (; j < nblk; ++j) {
        const int st = j % kStages;
        if (!mbar_wait(bar(kBarKvEmpty + st), ((j / kStages) & 1) ^ 1, p.err, ERR_WAIT_MMA))
          break;
        const uint32_t b = bar(kBarKvFull + st);
        const int kb = kb0 + j;
        mbar_expect_tx(b, kKBytes + kVBytes);
        tma_load_2d(base + kOffK + st * kKBytes, &tmK, b, 0, g * p.ring_pitch + kb * 128);
        tma_load_2d(base + kOffV + st * kVBytes, &tmV, b, kb * 128, g * kHeadDim);
        tma_load_2d(base + kOffV + st * kVBytes + kVSub, &tmV, b, kb * 128 + 64, g * kHeadDim);
      }
      // nothing may be in flight when the CTA exits
      mbar_wait(bar(kBarQ), 0, p.err, ERR_WAIT_TMA);
      for (int i = j - 1; i >= 0 && i >= j - kStages; --i)
        mbar_wait(bar(kBarKvFull + i % kStages), (i / kStages) & 1, p.err, ERR_WAIT_TMA);
    }
  } else if (warp == 9 || warp == 10) {
    // ------------------------------------------------------------ MMA issue for tile x
    // One issuing thread per tile, so neither tile's MMAs wait behind the other's events;
    // tcgen05.commit tracks only the MMAs of the thread that issues it.
    const int x = warp - 9;
    if (lane == 0 && aligned && nblk > 0) {
      const uint32_t idesc_s = idesc_bf16_f32(128, 128);
      const uint32_t idesc_o = idesc_f16_f32(128, 64);  // P and V^T are fp16
      // descriptors of the stage bases; K steps of 16 elements add 32 B (2 in the encoded
      // address field) inside the 128-byte swizzle atom
      const uint64_t dq = sdesc_k_sw128(base + kOffQ + x * kQBytes);
      const uint64_t dk0 = sdesc_k_sw128(base + kOffK);
      const uint64_t dv0 = sdesc_k_sw128(base + kOffV);
      const uint32_t s_tmem = tmem + kColS + 128u * x;
      const uint32_t p_tmem = tmem + kColP + 64u * x;
      const uint32_t o_tmem = tmem + kColO + 64u * x;
      auto issue_s = [&](int j) {  // S_X(j) = Q_X K_j^T
        const uint64_t dk = dk0 + static_cast<uint64_t>(((j % kStages) * kKBytes) >> 4);
#pragma unroll
        for (int k = 0; k < 4; ++k) mma_bf16_ss(s_tmem, dq + 2 * k, dk + 2 * k, idesc_s, k != 0);
        mma_commit(bar(kBarS + x));
      };
      bool ok = mbar_wait(bar(kBarQ), 0, p.err, ERR_WAIT_TMA) &&
                mbar_wait(bar(kBarKvFull), 0, p.err, ERR_WAIT_TMA);
      tc_fence_after();
      if (ok) issue_s(0);
      for (int j = 0; j < nblk && ok; ++j) {
        const int st = j % kStages;
        // S of the next block as soon as the softmax has read S(j)
        if (j + 1 < nblk) {
          ok = mbar_wait(bar(kBarKvFull + (j + 1) % kStages), ((j + 1) / kStages) & 1, p.err,
                         ERR_WAIT_TMA) &&
               mbar_wait(bar(kBarSFree + x), j & 1, p.err, ERR_WAIT_EPI);
          tc_fence_after();
          if (!ok) break;
          issue_s(j + 1);
        }
        // P V of this block once P(j) is written
        ok = mbar_wait(bar(kBarP + x), j & 1, p.err, ERR_WAIT_EPI);
        tc_fence_after();
        if (!ok) break;
        const uint64_t dv = dv0 + static_cast<uint64_t>((st * kVBytes) >> 4);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          mma_bf16_ts(o_tmem, p_tmem + 8u * kk,
                      dv + static_cast<uint64_t>((((kk >> 2) * kVSub) >> 4) + 2 * (kk & 3)),
                      idesc_o, (j | kk) != 0);
        mma_commit(bar(kBarPv + x));
        mma_commit(bar(kBarKvEmpty + st));  // one of the two arrivals that free the stage
      }
      mma_commit(bar(kBarDone + x));
      mbar_wait(bar(kBarDone + x), 0, p.err, ERR_WAIT_MMA);
    }
  } else {
    // ------------------------------------------------------------ softmax, tile x
    const int x = warp >> 2;
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t s_col = tmem + lane_off + kColS + 128u * x;
    const uint32_t p_col = tmem + lane_off + kColP + 64u * x;
    const uint32_t o_col = tmem + lane_off + kColO + 64u * x;
    const float sl2 = p.scale_log2;
    float m_used = -INFINITY, l_run = 0.f;
    bool ok = aligned;
    for (int j = 0; j < nblk && ok; ++j) {
      const bool got = mbar_wait(bar(kBarS + x), j & 1, p.err, ERR_WAIT_MMA);
      if (!__all_sync(0xffffffffu, got)) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t sr[4][32];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld_32x32b_x32(s_col + 32 * c, sr[c]);
      tmem_ld_wait();
      tc_fence_before();
      mbar_arrive(bar(kBarSFree + x));  // S_X may now receive the next block's scores
      const int valid = n_keys - (kb0 + j) * 128;
      if (valid < 128) {  // ragged last key block (warp-uniform branch)
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (32 * c + e >= valid) sr[c][e] = 0xff800000u;  // -inf
      }
      // row max: 8 independent chains of 16 elements, then a short tree
      float m8[8];
#pragma unroll
      for (int q8 = 0; q8 < 8; ++q8) {
        const uint32_t* v = sr[q8 >> 1] + 16 * (q8 & 1);
        float m = __uint_as_float(v[0]);
#pragma unroll
        for (int e = 1; e < 15; e += 2)
          m = fmax3(m, __uint_as_float(v[e]), __uint_as_float(v[e + 1]));
        m8[q8] = fmaxf(m, __uint_as_float(v[15]));
      }
      const float mx = fmax3(fmax3(m8[0], m8[1], m8[2]), fmax3(m8[3], m8[4], m8[5]),
                             fmaxf(m8[6], m8[7]));
      const float mb = mx * sl2;
      const bool grow = mb > m_used + kRescaleLog2;
      const float m_new = grow ? mb : m_used;
      // P = exp2(s * scale - m) in fp16 pairs: one packed FMA, one rounding to fp16 and one
      // packed ex2 per two keys; the row sum is a pairwise fp16x2 tree per 64 keys (sums stay
      // below 2^15 because P <= 2^8) added into fp32. This runs while the tensor core may
      // still be reading P_X(j-1): only the store of P(j) and the rescale of O wait for it.
      // Warp q of tile 0 and warp q of tile 1 share one SMSP, whose conversion and ex2 units
      // bound this loop. They take turns on the exponentials (tile 0 block j, tile 1 block j,
      // tile 0 block j+1, ...), so each one's S load, P V wait and P store run while the other
      // computes instead of both stalling at once.
      if (x == 1 || j > 0) {
        const bool turn = mbar_wait(bar(kBarTurn + 4 * x + quarter), (x == 1 ? j : j - 1) & 1,
                                    p.err, ERR_WAIT_EPI);
        if (!__all_sync(0xffffffffu, turn)) {
          ok = false;
          break;
        }
      }
      const uint64_t sc2 = pack_f32x2(sl2, sl2);
      const uint64_t ng2 = pack_f32x2(-m_new, -m_new);
      float lsum = 0.f;
      uint32_t pk[2][32];
#pragma unroll
      for (int half = 0; half < 2; ++half) {
#pragma unroll
        for (int cc = 0; cc < 2; ++cc)
#pragma unroll
          for (int e = 0; e < 32; e += 2)
            pk[half][cc * 16 + (e >> 1)] =
                exp2_pair_f16(__uint_as_float(sr[2 * half + cc][e]),
                              __uint_as_float(sr[2 * half + cc][e + 1]), sc2, ng2);
        uint32_t t16[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) t16[i] = hadd2(pk[half][2 * i], pk[half][2 * i + 1]);
#pragma unroll
        for (int stride = 8; stride > 0; stride >>= 1)
#pragma unroll
          for (int i = 0; i < stride; ++i) t16[i] = hadd2(t16[i], t16[i + stride]);
        lsum += f16x2_sum(t16[0]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(kBarTurn + 4 * (1 - x) + quarter));
      // P_X and O_X are free once the P V of the previous block has completed
      if (j > 0) {
        const bool pv = mbar_wait(bar(kBarPv + x), (j - 1) & 1, p.err, ERR_WAIT_MMA);
        if (!__all_sync(0xffffffffu, pv)) {
          ok = false;
          break;
        }
        tc_fence_after();
      }
      if (grow && j > 0) l_run *= ex2_approx(m_used - m_new);
      if (__any_sync(0xffffffffu, grow && j > 0)) {
        const float f = (grow && j > 0) ? ex2_approx(m_used - m_new) : 1.0f;
#pragma unroll 1
        for (int c = 0; c < 64; c += 16) {
          uint32_t o0[16];
          tmem_ld_32x32b_x16(o_col + c, o0);
          tmem_ld_wait();
#pragma unroll
          for (int d = 0; d < 16; ++d) o0[d] = __float_as_uint(__uint_as_float(o0[d]) * f);
          tmem_st_32x32b_x16(o_col + c, o0);
        }
      }
      m_used = m_new;
      tmem_st_32x32b_x32(p_col, pk[0]);
      tmem_st_32x32b_x32(p_col + 32, pk[1]);
      l_run += lsum;
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(bar(kBarP + x));
    }
    // ------------------------------------------------------------ output of tile x
    float o[64];
#pragma unroll
    for (int d = 0; d < 64; ++d) o[d] = 0.f;
    if (ok && nblk > 0) {
      const bool got = mbar_wait(bar(kBarPv + x), (nblk - 1) & 1, p.err, ERR_WAIT_MMA);
      ok = __all_sync(0xffffffffu, got);
      if (ok) {
        tc_fence_after();
        uint32_t o0[32], o1[32];
        tmem_ld_32x32b_x32(o_col, o0);
        tmem_ld_32x32b_x32(o_col + 32, o1);
        tmem_ld_wait();
#pragma unroll
        for (int d = 0; d < 32; ++d) {
          o[d] = __uint_as_float(o0[d]);
          o[32 + d] = __uint_as_float(o1[d]);
        }
      }
    }
    const int rho = (2 * blockIdx.x + x) * kBM + row;
    const int hl = rho / p.lq_pad;
    const int r = rho - hl * p.lq_pad;
    if (ok && hl < hpg && r < p.Lq) {
      const int h = g * hpg + hl;
      if (p.splits == 1) {
        const float inv = 1.0f / l_run;
        uint4* dst = reinterpret_cast<uint4*>(p.out + static_cast<size_t>(r) * p.ld_out +
                                              h * kHeadDim);
#pragma unroll
        for (int k = 0; k < 8; ++k)
          dst[k] = make_uint4(pack_bf16x2(o[8 * k] * inv, o[8 * k + 1] * inv),
                              pack_bf16x2(o[8 * k + 2] * inv, o[8 * k + 3] * inv),
                              pack_bf16x2(o[8 * k + 4] * inv, o[8 * k + 5] * inv),
                              pack_bf16x2(o[8 * k + 6] * inv, o[8 * k + 7] * inv));
      } else {
        const size_t idx = (static_cast<size_t>(blockIdx.z) * p.heads + h) * p.Lq + r;
        float4* dst = reinterpret_cast<float4*>(p.part_o + idx * kHeadDim);
#pragma unroll
        for (int k = 0; k < 16; ++k)
          dst[k] = make_float4(o[4 * k], o[4 * k + 1], o[4 * k + 2], o[4 * k + 3]);
        reinterpret_cast<float2*>(p.part_ml)[idx] =
            make_float2(nblk > 0 ? m_used : -INFINITY, l_run);
      }
    }
  }

  grid_dep_launch();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// One warp per (row, head): O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s.
__global__ void attn_combine_kernel(const float* __restrict__ part_o,
                                    const float* __restrict__ part_ml, int splits, int Lq,
                                    int heads, __nv_bfloat16* __restrict__ out, int ld_out) {
  grid_dep_wait();
  grid_dep_launch();
  const int wid = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (wid >= Lq * heads) return;
  const int r = wid / heads, h = wid - r * heads;
  const float2* ml = reinterpret_cast<const float2*>(part_ml);
  float M = -INFINITY;
  for (int s = 0; s < splits; ++s)
    M = fmaxf(M, ml[(static_cast<size_t>(s) * heads + h) * Lq + r].x);
  float a0 = 0.f, a1 = 0.f, l = 0.f;
  for (int s = 0; s < splits; ++s) {
    const size_t idx = (static_cast<size_t>(s) * heads + h) * Lq + r;
    const float2 v = ml[idx];
    const float w = ex2_approx(v.x - M);
    l = fmaf(w, v.y, l);
    const float2 o = reinterpret_cast<const float2*>(part_o + idx * kHeadDim)[lane];
    a0 = fmaf(w, o.x, a0);
    a1 = fmaf(w, o.y, a1);
  }
  const float inv = 1.0f / l;
  reinterpret_cast<uint32_t*>(out + static_cast<size_t>(r) * ld_out + h * kHeadDim)[lane] =
      pack_bf16x2(a0 * inv, a1 * inv);
}

int attention_splits(int units, int nblk, int num_sms) {
  int best = 1;
  long long best_cost = -1;
  for (int s = 1; s <= 4; ++s) {
    const long long ctas = static_cast<long long>(units) * s;
    const long long waves = (ctas + num_sms - 1) / num_sms;
    const long long cost = waves * ((nblk + s - 1) / s) * 100 + (s > 1 ? 150 : 0);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = s;
    }
  }
  return best;
}

cudaError_t launch_attention(const CUtensorMap& tmQ, const CUtensorMap& tmQ8,
                             const CUtensorMap& tmK,
                             const CUtensorMap& tmVt, const AttnParams& p, cudaStream_t s) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         attn::kSmem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const int tiles = attention_tiles_per_group(p.Lq, p.heads, p.groups);
  const dim3 grid((tiles + 1) / 2, p.groups, p.splits);
  cudaError_t e = launch_pdl(attn_kernel, grid, dim3(attn::kThreads), attn::kSmem, s, tmQ, tmQ8, tmK,
                             tmVt, p);
  if (e != cudaSuccess || p.splits == 1) return e;
  const long long warps = static_cast<long long>(p.Lq) * p.heads;
  return launch_pdl(attn_combine_kernel, dim3(static_cast<int>((warps + 7) / 8)), dim3(256), 0,
                    s, static_cast<const float*>(p.part_o), static_cast<const float*>(p.part_ml),
                    p.splits, p.Lq, p.heads, p.out, p.ld_out);
}

}  // namespace fd
