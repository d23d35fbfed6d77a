// tcgen05 / TMEM bf16 GEMM with fused epilogues: out = epilogue(A W^T + bias).
//
// A: bf16 [M][K] row-major (activations), W: bf16 [N][K] row-major (nn.Linear weight), both
// K-major, loaded by TMA with the 128-byte swizzle into a ring of shared-memory stages.
// One persistent CTA per SM walks 128 x BN output tiles. Warp roles:
//   warp 0 (one lane)  TMA producer: stages of 128x64 (A) and BNx64 (W)
//   warp 1 (one lane)  MMA issuer: 4 x tcgen05.mma (K = 16 each) per stage into a TMEM
//                      accumulator; two accumulators so the epilogue of tile i overlaps the
//                      MMAs of tile i+1
//   warps 2-5          epilogue: each thread owns one accumulator row (TMEM lane), applies
//                      the fused epilogue, and writes its row of a 32-row slab into a
//                      128-byte-swizzled staging buffer; one lane then stores the slab with a
//                      TMA bulk tensor store (a bulk reduce-add for the residual), so global
//                      writes are whole lines and rows past M are clipped by the tensor map
// Fused epilogues (the linear layers of Sec. 3.2 / 3.4 and Eq. projection / temporal_upsample):
//   EPI_F32    out = acc + b                    (patch-embed, head layer 2)
//   EPI_RESID  h  += acc + b                    (out-projection, MLP layer 2: residual)
//   EPI_GELU   out = bf16(GELU(acc + b))        (MLP layer 1, head layer 1)
//   EPI_TUP    channel block tau of token l -> refined token tau*L + l   (Eq. temporal_upsample)
//   EPI_SWIGLU out = bf16(SiLU(gate + b) * (up + b)) (gated MLP layer 1 of the XL layout; gate
//              and up rows interleaved in blocks of 32, so 128 columns give 64 outputs)
//   EPI_GELU_F8 out = e4m3(GELU(acc s_col + b) s_out)  (FP8 MLP layer 1, Sec. 4.6)
//   EPI_SWIGLU_F8 out = e4m3(SiLU(gate) up s_out), gate / up = acc s_col + b in the interleaved
//              blocks of EPI_SWIGLU (the FP8 gated MLP layer 1; 256 columns -> 128 outputs)
// FP8 operands (p.fp8): A and W are e4m3 with a K-block of 128 elements (the same 128-byte
// swizzled rows), tcgen05.mma kind::f8f6f4 with K = 32 per instruction; the fp32 epilogues
// then scale the accumulator per column by s_A s_W[n] (p.col_scale).
//   EPI_QKV    bias; KV-norm (RMS over D_h) on K and V (or QK-norm on Q and K); 3D-RoPE on Q
//              and K; Q to its buffer,
//              K (bf16) and V (transposed, fp16) into ring slot t mod W of the layer's cache
//              (Sec. 3.3)
//
// This header holds the kernel template and its launcher; fd_gemm.cu instantiates the
// instances of every epilogue but EPI_QKV, fd_gemm_qkv.cu those of EPI_QKV (compiled in
// parallel, and the QKV epilogue's code does not weigh on the others' register allocation).
#pragma once
#include "fd_internal.h"
#include "fd_ptx.cuh"

namespace fd {

// PAIR: the tile is 256 x BN, computed by a cluster of two CTAs with tcgen05 cta_group::2
// MMAs issued by the even CTA: each CTA holds its 128 rows of A and half (BN/2 rows) of W per
// stage, the pair's tensor cores read both halves, and each CTA's TMEM receives its 128 rows of
// the accumulator. Per SM, a stage then needs 16 KB + 64 BN bytes for 2 BN MMA cycles instead of
// 16 KB + 128 BN, which is what bounds the single-CTA kernel (shared-memory intake per SM).
template <int BN, bool PAIR>
struct GemmCfg {
  static constexpr int kABytes = kBM * kBK * 2;  // 16 KB
  static constexpr int kBRows = PAIR ? BN / 2 : BN;
  static constexpr int kBBytes = kBRows * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kRoom = (227 * 1024 - 4 * 2 * 4096 - 256) / kStageBytes;
  static constexpr int kStages = PAIR ? (kRoom > 8 ? 8 : kRoom) : (BN >= 192 ? 4 : 6);
  static constexpr int kTmemCols = 2 * BN <= 128 ? 128 : (2 * BN <= 256 ? 256 : 512);
  static constexpr int kStgOffset = kStages * kStageBytes;   // 4 warps x 2 x 4 KB staging
  static constexpr int kBarOffset = kStgOffset + 4 * 2 * 4096;
  static constexpr int kSmem = kBarOffset + 256;
  static_assert(kSmem <= 227 * 1024, "shared memory");
  static_assert((kBRows * 128) % 1024 == 0, "W stages start on a swizzle atom");
};

// one 128-byte row (8 x 16 B) of a 32-row slab in the 128-byte-swizzled layout of a TMA box
__device__ __forceinline__ void put_row_sw128(uint8_t* buf, int row, const uint32_t* w) {
#pragma unroll
  for (int k = 0; k < 8; ++k)
    *reinterpret_cast<uint4*>(buf + row * 128 + ((k ^ (row & 7)) << 4)) =
        make_uint4(w[4 * k], w[4 * k + 1], w[4 * k + 2], w[4 * k + 3]);
}

// 1 + erf(a), after Abramowitz & Stegun, Handbook of Mathematical Functions, formula 7.1.26:
// for b = |a|, erf(b) = 1 - (a1 t + a2 t^2 + a3 t^3 + a4 t^4 + a5 t^5) e^(-b^2) with
// t = 1 / (1 + p b), absolute error at most 1.5e-7. With E = the polynomial times e^(-b^2),
// 1 + erf(a) = 2 - E for a >= 0 and E for a < 0 (erf is odd), so the negative side has no
// cancellation. In fp32 with the hardware reciprocal and exp2 (a few ulp each) the error stays
// near 1e-7, far below the bf16 (2^-9) and e4m3 (2^-4) rounding of the GELU outputs.
__device__ __forceinline__ float one_plus_erf(float a) {
  const float b = fabsf(a);
  float t;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(t) : "f"(fmaf(0.3275911f, b, 1.0f)));
  float y = fmaf(1.061405429f, t, -1.453152027f);
  y = fmaf(y, t, 1.421413741f);
  y = fmaf(y, t, -0.284496736f);
  y = fmaf(y, t, 0.254829592f);
  const float e = y * t * ex2_approx(-(b * b) * 1.44269504088896341f);  // erfc(b)
  return a >= 0.f ? 2.0f - e : e;
}

// GELU, exact (erf) form: x Phi(x) = 0.5 x (1 + erf(x / sqrt 2))
__device__ __forceinline__ float gelu_erf(float x) {
  return 0.5f * x * one_plus_erf(x * 0.70710678118654752f);
}

// 32 consecutive fp32 values (16-byte aligned) as eight vector loads; the same for every lane
__device__ __forceinline__ void load32(const float* p, float (&v)[32]) {
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const float4 q = __ldg(reinterpret_cast<const float4*>(p) + k);
    v[4 * k] = q.x;
    v[4 * k + 1] = q.y;
    v[4 * k + 2] = q.z;
    v[4 * k + 3] = q.w;
  }
}

// SiLU(x) = x / (1 + e^-x) with the fast division (a few ulp; for x -> -inf the denominator
// overflows and the quotient goes to 0, the correct limit)
__device__ __forceinline__ float silu(float x) { return __fdividef(x, 1.0f + __expf(-x)); }

// cos / sin of the 32 rotation pairs of one token (3D-RoPE: temporal pairs first, then row,
// then column; angle = position * base^(-2i/d_band)). Temporal values come from the chunk's
// table (fp64-evaluated, any stream length); row / column angles are below 2^12 rad, reduced to
// [-pi, pi] in fp32 (2 pi split in two parts) and evaluated with the fast sin / cos.
__device__ __forceinline__ void rope_table(const QkvEpi& q, const float2* rope_t, int tau, int y,
                                           int x, float* c, float* s) {
#pragma unroll
  for (int i = 0; i < kRopePairs; ++i) {
    if (i < q.band_t) {
      const float2 v = __ldcg(rope_t + tau * q.band_t + i);
      c[i] = v.x;
      s[i] = v.y;
    } else {
      const int pos = i < q.band_t + q.band_s ? y : x;
      const float a = static_cast<float>(pos) * q.inv_freq_s[i];
      const float k = rintf(a * 0.159154943091895336f);
      float r = fmaf(-k, 6.28318548202514648f, a);
      r = fmaf(-k, -1.74845553e-7f, r);
      __sincosf(r, &s[i], &c[i]);
    }
  }
}

// QKV: 0 for every epilogue but EPI_QKV (no QKV code), 1 for EPI_QKV on one stream, 2 for
// EPI_QKV on stacked streams (q.streams > 0).
// DS (single CTAs, K = 64): the attention's scores backward. Each tile holds two products, S =
// Q K^T (tmA, tmB) and dP = dO V^T (tmK, tmV: A and B of the second product), one K block each,
// in two TMEM accumulators; the epilogue turns them into dS = P (dP - delta) scale with P =
// exp(S scale - lse) (p.ds), written as dS rows and dS^T, P^T columns (bf16). S and dP are never
// stored.
template <int BN, bool PAIR, int QKV, bool DS = false>
__global__ void __launch_bounds__(192, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmO, const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const __grid_constant__ GemmParams p) {
  using C = GemmCfg<BN, PAIR>;
  // accumulator columns of one tile (DS: S and dP side by side), two tiles in flight
  constexpr uint32_t kAccCols = DS ? 2 * BN : BN;
  constexpr int kTmemCols = DS ? 4 * BN : C::kTmemCols;
  static_assert(!DS || (!PAIR && QKV == 0 && 4 * BN <= 512), "scores backward: single CTAs");
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kBarOffset);
  const uint32_t bar_full = smem_u32(bars);                    // [kStages]
  const uint32_t bar_empty = smem_u32(bars + C::kStages);      // [kStages]
  const uint32_t bar_tfull = smem_u32(bars + 2 * C::kStages);  // [2]
  const uint32_t bar_tempty = smem_u32(bars + 2 * C::kStages + 2);  // [2]
  const uint32_t bar_done = smem_u32(bars + 2 * C::kStages + 4);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * C::kStages + 5);
  const uint32_t sA = smem_u32(smem);
  const uint32_t sB = sA + C::kStages * C::kABytes;
  const bool aligned = (sA & 1023u) == 0;

  // CTA pairs: rank 0 issues the MMAs; every load of the pair completes on rank 0's full
  // barrier; the MMA commits arrive in both CTAs (stage release, accumulator ready); both CTAs'
  // epilogue warps release the accumulator on rank 0's barrier
  const uint32_t rank = PAIR ? cluster_ctarank() : 0;
  const int tile_rows = PAIR ? 2 * kBM : kBM;
  const int m_tiles = (p.M + tile_rows - 1) / tile_rows;
  const int n_tiles = (p.N + BN - 1) / BN;
  const int tiles = m_tiles * n_tiles;
  const int cta0 = PAIR ? static_cast<int>(blockIdx.x) / 2 : static_cast<int>(blockIdx.x);
  const int ctas = PAIR ? static_cast<int>(gridDim.x) / 2 : static_cast<int>(gridDim.x);
  const int kel = p.fp8 ? 2 * kBK : kBK;  // K elements per 128-byte stage row
  const int nk = DS ? 2 : (p.K + kel - 1) / kel;  // DS: the two products' K blocks
  const uint32_t full_tx = PAIR ? 2 * C::kStageBytes : C::kStageBytes;  // on rank 0's barrier
  const uint32_t bar_full0 = PAIR ? mapa_rank(bar_full, 0) : bar_full;
  auto load = [&](uint32_t dst, const CUtensorMap* m, int s, int x, int y) {
    if (PAIR) tma_load_2d_pair(dst, m, bar_full0 + 8 * s, x, y);
    else tma_load_2d(dst, m, bar_full + 8 * s, x, y);
  };

  if (threadIdx.x == 0) {
    if (!aligned) atomicOr(p.err, ERR_SMEM_ALIGN);
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(bar_tfull + 8 * a, 1);
      mbar_init(bar_tempty + 8 * a, PAIR ? 8 : 128);  // pairs: one arrive per epilogue warp
    }
    mbar_init(bar_done, 1);
    fence_barrier_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
  }
  if (PAIR) cluster_sync();  // both CTAs' barriers exist before any load or commit reaches them
  // Weights that no kernel of the stream writes (p.w_static) are loaded into the first stages
  // while the previous kernel is still finishing; only the activations wait for it. Thread 0
  // is the TMA producer and initialised the barriers above.
  const int pre = (p.w_static && aligned && cta0 < tiles)
                      ? (nk < C::kStages ? nk : C::kStages)
                      : 0;
  if (threadIdx.x == 0) {
    const int nb0 = (cta0 % n_tiles) * BN + static_cast<int>(rank) * C::kBRows;
    for (int kb = 0; kb < pre; ++kb) {
      if (rank == 0) mbar_expect_tx(bar_full + 8 * kb, full_tx);
      load(sB + kb * C::kBBytes, &tmB, kb, kb * kel, nb0);
    }
  }
  grid_dep_wait();  // inputs written by the previous kernel; TMEM freed by its CTAs
  if (warp == 1) {
    if (PAIR) {
      tmem_alloc_pair(smem_u32(tmem_slot), kTmemCols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(smem_u32(tmem_slot), kTmemCols);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (aligned && warp == 0 && lane == 0) {
    // ------------------------------------------------------------ TMA producer
    int it = 0;
    bool ok = true;
    for (int tile = cta0; tile < tiles && ok; tile += ctas) {
      const int m0 = (tile / n_tiles) * tile_rows + static_cast<int>(rank) * kBM;
      const int nb0 = (tile % n_tiles) * BN + static_cast<int>(rank) * C::kBRows;
      for (int kb = 0; kb < nk; ++kb, ++it) {
        const int s = it % C::kStages;
        const uint32_t ph = (it / C::kStages) & 1;
        if (it < pre) {  // W already on its way: the activation half of the stage
          load(sA + s * C::kABytes, &tmA, s, kb * kel, m0);
          continue;
        }
        if (!mbar_wait(bar_empty + 8 * s, ph ^ 1, p.err, ERR_WAIT_MMA)) { ok = false; break; }
        if (rank == 0) mbar_expect_tx(bar_full + 8 * s, full_tx);
        if (DS) {  // block 0: Q and K; block 1: dO and V (K = 64, one block each)
          load(sA + s * C::kABytes, kb == 0 ? &tmA : &tmK, s, 0, m0);
          load(sB + s * C::kBBytes, kb == 0 ? &tmB : &tmV, s, 0, nb0);
          continue;
        }
        load(sA + s * C::kABytes, &tmA, s, kb * kel, m0);
        load(sB + s * C::kBBytes, &tmB, s, kb * kel, nb0);
      }
    }
    // drain: the loads issued last must land before the CTA may exit (pairs: they have once
    // rank 0's MMAs have read their stages, which releases the stage in both CTAs)
    for (int j = it - 1; j >= 0 && j >= it - C::kStages; --j) {
      if (PAIR)
        mbar_wait(bar_empty + 8 * (j % C::kStages), (j / C::kStages) & 1, p.err, ERR_WAIT_MMA);
      else
        mbar_wait(bar_full + 8 * (j % C::kStages), (j / C::kStages) & 1, p.err, ERR_WAIT_TMA);
    }
  } else if (aligned && warp == 1 && rank == 0) {
    // ------------------------------------------------------------ MMA issuer
    // (the whole warp runs the loop; one elected lane issues)
    const uint32_t idesc =
        p.fp8 ? idesc_e4m3_f32(tile_rows, BN) : idesc_bf16_f32(tile_rows, BN);
    int it = 0, tc = 0;
    bool ok = true;
    for (int tile = cta0; tile < tiles && ok; tile += ctas, ++tc) {
      const int acc = tc & 1;
      if (!mbar_wait_warp(bar_tempty + 8 * acc, ((tc >> 1) & 1) ^ 1, p.err, ERR_WAIT_EPI))
        break;
      tc_fence_after();
      const uint32_t d_acc = tmem + static_cast<uint32_t>(acc) * kAccCols;
      for (int kb = 0; kb < nk; ++kb, ++it) {
        // DS: each K block is its own product, in its own accumulator
        const uint32_t d_tmem = DS ? d_acc + static_cast<uint32_t>(kb) * BN : d_acc;
        const int kacc = DS ? 0 : kb;  // accumulate over K blocks (DS: within the block only)
        const int s = it % C::kStages;
        if (!mbar_wait_warp(bar_full + 8 * s, (it / C::kStages) & 1, p.err, ERR_WAIT_TMA)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = sA + s * C::kABytes;
        const uint32_t b0 = sB + s * C::kBBytes;
        // one 128-byte row of the stage: 4 MMAs of K = 16 bf16 (or 32 e4m3) elements
        static_assert(kBK == 64, "a K block is one 128-byte swizzle row of bf16");
        const uint64_t da = sdesc_k_sw128(a0), db = sdesc_k_sw128(b0);
        if (p.fp8) {
          if (PAIR) mma4_e4m3_ss_pair_w(d_tmem, da, db, idesc, kb != 0);
          else mma4_e4m3_ss_w(d_tmem, da, db, idesc, kb != 0);
        } else {
          if (PAIR) mma4_bf16_ss_pair_w(d_tmem, da, db, idesc, kacc != 0);
          else mma4_bf16_ss_w(d_tmem, da, db, idesc, kacc != 0);
        }
        // stage s free (in both CTAs of a pair) once these MMAs have read it
        if (PAIR) mma_commit_pair_w(bar_empty + 8 * s, 3);
        else mma_commit_w(bar_empty + 8 * s);
      }
      if (ok) {
        if (PAIR) mma_commit_pair_w(bar_tfull + 8 * acc, 3);
        else mma_commit_w(bar_tfull + 8 * acc);
      }
    }
    if (PAIR) mma_commit_pair_w(bar_done, 1);
    else mma_commit_w(bar_done);
    mbar_wait_warp(bar_done, 0, p.err, ERR_WAIT_MMA);
  } else if (aligned && warp >= 2) {
    // ------------------------------------------------------------ epilogue
    const int quarter = warp & 3;  // TMEM lanes this warp may read
    const int rloc = quarter * 32 + lane;
    uint8_t* stg = smem + C::kStgOffset + (warp - 2) * 8192;
    int sb = 0;
    // a free 4 KB staging buffer: the store issued from it two stores ago has read it
    auto acquire = [&]() -> uint8_t* {
      if (lane == 0) bulk_wait_read_1();
      __syncwarp();
      uint8_t* b = stg + sb * 4096;
      sb ^= 1;
      return b;
    };
    auto publish = [&]() {  // make the slab visible to the TMA engine
      fence_proxy_async_smem();
      __syncwarp();
    };
    if (lane == 0) {
      prefetch_tmap(&tmO);
      if (QKV) {
        prefetch_tmap(&tmK);
        if (p.v_tma) prefetch_tmap(&tmV);
      }
    }
    int t = 0;
    if (QKV) t = p.qkv.step_dev ? *p.qkv.step_dev : p.qkv.step_host;
    int tc = 0;
    const uint32_t bar_tempty0 = PAIR ? mapa_rank(bar_tempty, 0) : bar_tempty;
    for (int tile = cta0; tile < tiles; tile += ctas, ++tc) {
      const int acc = tc & 1;
      const int m0 = (tile / n_tiles) * tile_rows + static_cast<int>(rank) * kBM;
      const int n0 = (tile % n_tiles) * BN;
      const int row0 = m0 + quarter * 32;  // first row of this warp's slab
      const int row = m0 + rloc;
      const bool row_ok = row < p.M;
      const uint32_t tbase =
          tmem + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(acc) * kAccCols;
      // The tile's bias (and column-scale) lines go into L1 while its MMAs still run, so the
      // per-chunk loads below do not each wait a round trip to L2 after the accumulator is ready.
      if (!DS && lane < BN / 32 && n0 + 32 * lane < p.N) {
        prefetch_l1(p.bias + n0 + 32 * lane);
        if (p.col_scale != nullptr) prefetch_l1(p.col_scale + n0 + 32 * lane);
      }
      // wait for the tile's accumulator; all lanes leave together (TMEM loads are collective)
      auto acc_ready = [&]() -> bool {
        const bool got = mbar_wait(bar_tfull + 8 * acc, (tc >> 1) & 1, p.err, ERR_WAIT_MMA);
        if (!__all_sync(0xffffffffu, got)) return false;
        tc_fence_after();
        return true;
      };
      if (!QKV && !acc_ready()) break;

      if (QKV) {
        const QkvEpi& q = p.qkv;
        float rc[kRopePairs], rsn[kRopePairs];  // identity rotation for rows past M / padding
#pragma unroll
        for (int i = 0; i < kRopePairs; ++i) {
          rc[i] = 1.0f;
          rsn[i] = 0.0f;
        }
        const int rows_chunk = q.frames_per_chunk * q.tokens;  // = M (single stream)
        int slot = t % q.window;
        // batched: this row's stream, frame and token, its ring row (or -1 for padding)
        int ring_row = -1;
        __nv_bfloat16* k_ring = q.k_ring;
        __half* vt_ring = q.vt_ring;
        if (QKV == 2) {
          const int si = row / q.stream_rows, loc = row - si * q.stream_rows;
          const int tau = loc / q.frame_rows, l = loc - tau * q.frame_rows;
          if (row_ok && si < q.streams && l < q.tokens) {
            const QkvStream st = q.stream[si];
            slot = *st.step_dev % q.window;
            ring_row = slot * rows_chunk + tau * q.tokens + l;
            k_ring = st.k_ring;
            vt_ring = st.vt_ring;
            rope_table(q, st.rope_t, tau, l / q.grid_w, l % q.grid_w, rc, rsn);
          }
        } else if (row_ok) {
          const int l = row % q.tokens;
          rope_table(q, q.rope_t, row / q.tokens, l / q.grid_w, l % q.grid_w, rc, rsn);
          ring_row = slot * rows_chunk + row;
        }
        if (lane < 2) {  // the per-head norm gains (64 floats each)
          if (q.knorm_g != nullptr) prefetch_l1(q.knorm_g + 32 * lane);
          if (q.vnorm_g != nullptr) prefetch_l1(q.vnorm_g + 32 * lane);
        }
        // the rotation and ring position above depend only on the row: computed while the
        // MMAs of the tile still run
        if (!acc_ready()) break;
#pragma unroll 1
        for (int c = 0; c < BN; c += 64) {
          const int col = n0 + c;
          if (col >= p.N) break;  // warp-uniform
          uint32_t r0[32], r1[32];
          __syncwarp();  // tcgen05.ld is warp-collective: reconverge first
          tmem_ld_32x32b_x32(tbase + c, r0);
          tmem_ld_32x32b_x32(tbase + c + 32, r1);
          tmem_ld_wait();
          float v[64];
          {
            float b0[32], b1[32];
            load32(p.bias + col, b0);
            load32(p.bias + col + 32, b1);
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              v[j] = __uint_as_float(r0[j]) + b0[j];
              v[32 + j] = __uint_as_float(r1[j]) + b1[j];
            }
          }
          const int hidx = col / kHeadDim;
          const bool is_q = hidx < q.heads;
          const bool is_k = !is_q && hidx < q.heads + q.groups;
          if (q.qk_norm ? (is_q || is_k) : !is_q) {  // per-head RMSNorm, learned gain
            float ss = 0.f;
#pragma unroll
            for (int j = 0; j < 64; ++j) ss = fmaf(v[j], v[j], ss);
            const float rs = rsqrtf(ss * (1.0f / 64.0f) + q.eps);
            const float* g = is_k ? q.knorm_g : q.vnorm_g;
#pragma unroll
            for (int j = 0; j < 64; ++j) v[j] = v[j] * rs * __ldg(g + j);
          }
          if (is_q || is_k) {  // 3D-RoPE on interleaved pairs
#pragma unroll
            for (int i = 0; i < kRopePairs; ++i) {
              const float a = v[2 * i], b = v[2 * i + 1];
              v[2 * i] = a * rc[i] - b * rsn[i];
              v[2 * i + 1] = a * rsn[i] + b * rc[i];
            }
            uint32_t w[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) w[j] = pack_bf16x2(v[2 * j], v[2 * j + 1]);
            if (!is_q && QKV == 2) {  // batched: K row straight into its stream's ring
              if (ring_row >= 0) {
                uint4* dst = reinterpret_cast<uint4*>(
                    k_ring + (static_cast<size_t>(hidx - q.heads) * q.ring_pitch + ring_row) *
                                 kHeadDim);
#pragma unroll
                for (int k = 0; k < 8; ++k)
                  dst[k] = make_uint4(w[4 * k], w[4 * k + 1], w[4 * k + 2], w[4 * k + 3]);
              }
              continue;
            }
            uint8_t* buf = acquire();
            put_row_sw128(buf, lane, w);
            publish();
            if (lane == 0 && row0 < p.M) {  // a slab wholly past M stores nothing
              if (is_q) {
                tma_store_2d(&tmO, smem_u32(buf), hidx * kHeadDim, row0);
              } else {
                tma_store_4d(&tmK, smem_u32(buf), 0, row0, slot, hidx - q.heads);
              }
              bulk_commit();
            }
          } else if (p.v_tma && QKV != 2) {
            // V transposed: slab [64 dims][32 keys] fp16, stored into the ring's V^T slot view
            uint8_t* buf = acquire();
            __half* sv = reinterpret_cast<__half*>(buf);
#pragma unroll
            for (int j = 0; j < 64; ++j) sv[j * 32 + lane] = __float2half_rn(v[j]);
            publish();
            if (lane == 0 && row0 < p.M) {
              tma_store_4d(&tmV, smem_u32(buf), row0, slot, 0, hidx - q.heads - q.groups);
              bulk_commit();
            }
          } else if (ring_row >= 0) {  // V^T column by column (keys of a warp are adjacent)
            const int g = hidx - q.heads - q.groups;
            __half* dst = vt_ring + static_cast<size_t>(g) * kHeadDim * q.ring_pitch + ring_row;
#pragma unroll
            for (int j = 0; j < 64; ++j)
              dst[static_cast<size_t>(j) * q.ring_pitch] = __float2half_rn(v[j]);
          }
        }
      } else if (DS) {
        // scores backward of the tile: P = exp(S scale - lse) (0 on padding rows and keys),
        // dS = P (dP - delta) scale; dS rows (4 x 16 B per thread and chunk), dS^T and P^T
        // columns (one bf16 per lane and column: the warp's 32 rows are contiguous there)
        const DsEpi& q = p.ds;
        const bool live = row_ok && row % q.Pc % q.Lp < q.L;
        const float lse = row_ok ? __ldg(q.lse + row) : 0.f;
        const float dlt = row_ok ? __ldg(q.delta + row) : 0.f;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          const int col = n0 + c;
          if (col >= p.N) break;  // N % 32 == 0
          uint32_t rs[32], rp[32];
          __syncwarp();
          tmem_ld_32x32b_x32(tbase + c, rs);
          tmem_ld_32x32b_x32(tbase + BN + c, rp);
          tmem_ld_wait();
          if (!row_ok) continue;
          uint32_t dsw[16];
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            float pj[2], dj[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const bool key = (col + j + e) % q.Lp < q.L;
              pj[e] = live && key ? expf(__uint_as_float(rs[j + e]) * q.scale - lse) : 0.f;
              dj[e] = pj[e] * (__uint_as_float(rp[j + e]) - dlt) * q.scale;
            }
            dsw[j / 2] = pack_bf16x2(dj[0], dj[1]);
            const __nv_bfloat162 pb = __floats2bfloat162_rn(pj[0], pj[1]);
            const __nv_bfloat162 db = __floats2bfloat162_rn(dj[0], dj[1]);
            const size_t t0 = static_cast<size_t>(col + j) * p.M + row;
            q.PT[t0] = pb.x;
            q.PT[t0 + p.M] = pb.y;
            q.dST[t0] = db.x;
            q.dST[t0 + p.M] = db.y;
          }
          uint4* d = reinterpret_cast<uint4*>(q.dS + static_cast<size_t>(row) * p.N + col);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            d[k] = make_uint4(dsw[4 * k], dsw[4 * k + 1], dsw[4 * k + 2], dsw[4 * k + 3]);
        }
      } else if (p.epi == EPI_GELU) {
#pragma unroll 1
        for (int c = 0; c < BN; c += 64) {
          const int col = n0 + c;
          if (col >= p.N) break;
          uint32_t r0[32], r1[32];
          __syncwarp();
          tmem_ld_32x32b_x32(tbase + c, r0);
          tmem_ld_32x32b_x32(tbase + c + 32, r1);
          tmem_ld_wait();
          uint32_t w[32];
          {
            float b0[32], b1[32];
            load32(p.bias + col, b0);
            load32(p.bias + col + 32, b1);
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              w[j] = pack_bf16x2(gelu_erf(__uint_as_float(r0[2 * j]) + b0[2 * j]),
                                 gelu_erf(__uint_as_float(r0[2 * j + 1]) + b0[2 * j + 1]));
              w[16 + j] = pack_bf16x2(gelu_erf(__uint_as_float(r1[2 * j]) + b1[2 * j]),
                                      gelu_erf(__uint_as_float(r1[2 * j + 1]) + b1[2 * j + 1]));
            }
          }
          uint8_t* buf = acquire();
          put_row_sw128(buf, lane, w);
          publish();
          if (lane == 0 && row0 < p.M) {
            tma_store_2d(&tmO, smem_u32(buf), col, row0);
            bulk_commit();
          }
        }
      } else if (p.epi == EPI_GELU_F8) {
        // 128 accumulator columns -> one 128-byte row of e4m3 per slab
#pragma unroll 1
        for (int c = 0; c < BN; c += 128) {
          const int col = n0 + c;
          if (col >= p.N) break;
          uint32_t w[32];
#pragma unroll
          for (int q4 = 0; q4 < 4; ++q4) {
            uint32_t r[32];
            __syncwarp();
            tmem_ld_32x32b_x32(tbase + c + 32 * q4, r);
            tmem_ld_wait();
            const int cb = col + 32 * q4;
            float cs[32], bb[32];
            load32(p.col_scale + cb, cs);
            load32(p.bias + cb, bb);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              float f[4];
#pragma unroll
              for (int e = 0; e < 4; ++e)
                f[e] = gelu_erf(fmaf(__uint_as_float(r[4 * j + e]), cs[4 * j + e], bb[4 * j + e])) *
                       p.out_scale;
              w[8 * q4 + j] = pack_e4m3x4(f[0], f[1], f[2], f[3]);
            }
          }
          uint8_t* buf = acquire();
          put_row_sw128(buf, lane, w);
          publish();
          if (lane == 0 && row0 < p.M) {
            tma_store_2d(&tmO, smem_u32(buf), col, row0);
            bulk_commit();
          }
        }
      } else if (p.epi == EPI_SWIGLU_F8) {
        // 256 accumulator columns (4 blocks of 32 gate + 32 up) -> one 128-byte e4m3 row
#pragma unroll 1
        for (int c = 0; c < BN; c += 256) {
          const int col = n0 + c;
          if (col >= p.N) break;
          uint32_t w[32];
#pragma unroll
          for (int hh = 0; hh < 4; ++hh) {
            uint32_t rg[32], ru[32];
            __syncwarp();
            tmem_ld_32x32b_x32(tbase + c + 64 * hh, rg);
            tmem_ld_32x32b_x32(tbase + c + 64 * hh + 32, ru);
            tmem_ld_wait();
            const int cb = col + 64 * hh;
            float v[32];
            {
              float cs[32], bb[32];
              load32(p.col_scale + cb, cs);
              load32(p.bias + cb, bb);
#pragma unroll
              for (int j = 0; j < 32; ++j) v[j] = silu(fmaf(__uint_as_float(rg[j]), cs[j], bb[j]));
              load32(p.col_scale + cb + 32, cs);
              load32(p.bias + cb + 32, bb);
#pragma unroll
              for (int j = 0; j < 32; ++j)
                v[j] *= fmaf(__uint_as_float(ru[j]), cs[j], bb[j]) * p.out_scale;
            }
#pragma unroll
            for (int j = 0; j < 8; ++j)
              w[8 * hh + j] = pack_e4m3x4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
          }
          uint8_t* buf = acquire();
          put_row_sw128(buf, lane, w);
          publish();
          if (lane == 0 && row0 < p.M) {
            tma_store_2d(&tmO, smem_u32(buf), col / 2, row0);
            bulk_commit();
          }
        }
      } else if (p.epi == EPI_SWIGLU) {
#pragma unroll 1
        for (int c = 0; c < BN; c += 128) {
          const int col = n0 + c;
          if (col >= p.N) break;
          uint32_t w[32];
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            uint32_t rg[32], ru[32];
            __syncwarp();
            tmem_ld_32x32b_x32(tbase + c + 64 * hh, rg);
            tmem_ld_32x32b_x32(tbase + c + 64 * hh + 32, ru);
            tmem_ld_wait();
            float bgv[32], buv[32];
            load32(p.bias + col + 64 * hh, bgv);
            load32(p.bias + col + 64 * hh + 32, buv);
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              const float g0 = __uint_as_float(rg[2 * j]) + bgv[2 * j];
              const float g1 = __uint_as_float(rg[2 * j + 1]) + bgv[2 * j + 1];
              const float u0 = __uint_as_float(ru[2 * j]) + buv[2 * j];
              const float u1 = __uint_as_float(ru[2 * j + 1]) + buv[2 * j + 1];
              w[16 * hh + j] = pack_bf16x2(silu(g0) * u0, silu(g1) * u1);
            }
          }
          uint8_t* buf = acquire();
          put_row_sw128(buf, lane, w);
          publish();
          if (lane == 0 && row0 < p.M) {
            tma_store_2d(&tmO, smem_u32(buf), col / 2, row0);
            bulk_commit();
          }
        }
      } else if (BN == 256 && !PAIR && p.epi == EPI_PIXEL) {
        // head layer 2 with the pixel shuffle (Sec. 3.4 Step 3): each 32-column chunk of the
        // token's row is 32 / rs pixel rows of rs pixels, written as groups of 4 pixels
        const PixelEpi& px = p.pix;
        const int tau = row / px.tokens, l = row - tau * px.tokens;
        const bool out_row = row_ok && tau < px.frames;
        const int gy = l / px.gw, gx = l - gy * px.gw;
        const int rs = px.rs, rs2 = rs * rs, Wo = px.gw * rs, Ho = px.gh * rs;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          const int col = n0 + c;
          if (col >= p.N) break;
          uint32_t r[32];
          __syncwarp();
          tmem_ld_32x32b_x32(tbase + c, r);
          tmem_ld_wait();
          float bb[32];
          load32(p.bias + col, bb);
          if (!out_row) continue;
          const int ch = col / rs2, rem = col - ch * rs2;
#pragma unroll
          for (int j = 0; j < 32; j += 4) {
            const int y = gy * rs + (rem + j) / rs, x = gx * rs + (rem + j) % rs;
            const size_t o = ((static_cast<size_t>(ch) * px.frames + tau) * Ho + y) * Wo + x;
            const float v0 = __uint_as_float(r[j]) + bb[j];
            const float v1 = __uint_as_float(r[j + 1]) + bb[j + 1];
            const float v2 = __uint_as_float(r[j + 2]) + bb[j + 2];
            const float v3 = __uint_as_float(r[j + 3]) + bb[j + 3];
            if (px.u8) {
              *reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(px.out) + o) =
                  quant_u8(v0) | (quant_u8(v1) << 8) | (quant_u8(v2) << 16) |
                  (quant_u8(v3) << 24);
            } else {
              *reinterpret_cast<float4*>(static_cast<float*>(px.out) + o) =
                  make_float4(fminf(fmaxf(v0, -1.f), 1.f), fminf(fmaxf(v1, -1.f), 1.f),
                              fminf(fmaxf(v2, -1.f), 1.f), fminf(fmaxf(v3, -1.f), 1.f));
            }
          }
        }
      } else {  // EPI_F32, EPI_RESID, EPI_TUP: fp32 slabs of 32 columns
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          const int col = n0 + c;
          if (col >= p.N) break;
          uint32_t r[32];
          __syncwarp();
          tmem_ld_32x32b_x32(tbase + c, r);
          tmem_ld_wait();
          uint32_t w[32];
          float bb[32];
          load32(p.bias + col, bb);
          if (p.col_scale != nullptr) {  // FP8 operands: dequantise per column
            float cs[32];
            load32(p.col_scale + col, cs);
#pragma unroll
            for (int j = 0; j < 32; ++j)
              w[j] = __float_as_uint(fmaf(__uint_as_float(r[j]), cs[j], bb[j]));
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) w[j] = __float_as_uint(__uint_as_float(r[j]) + bb[j]);
          }
          uint8_t* buf = acquire();
          put_row_sw128(buf, lane, w);
          publish();
          if (lane == 0 && row0 < p.M) {
            if (p.epi == EPI_RESID) {
              tma_reduce_add_2d(&tmO, smem_u32(buf), col, row0);
            } else if (p.epi == EPI_TUP) {
              const int tau = col / p.tup_hidden;
              // rows stack streams of tup_tokens rows each: [stream][tau][token][channel]
              tma_store_4d(&tmO, smem_u32(buf), col - tau * p.tup_hidden, row0 % p.tup_tokens,
                           tau, row0 / p.tup_tokens);
            } else {
              tma_store_2d(&tmO, smem_u32(buf), col, row0);
            }
            bulk_commit();
          }
        }
      }
      __syncwarp();
      tc_fence_before();
      if (PAIR) {  // one arrive per warp on rank 0's barrier
        if (lane == 0) mbar_arrive_remote(bar_tempty0 + 8 * acc);
      } else {
        mbar_arrive(bar_tempty + 8 * acc);
      }
    }
    if (lane == 0) bulk_wait_all();  // every store has landed before the CTA exits
    __syncwarp();
  }
  grid_dep_launch();
  tc_fence_before();
  // pairs: neither CTA leaves (or frees the TMEM columns both hold) before the other is done
  if (PAIR) cluster_sync();
  else __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if (PAIR) tmem_dealloc_pair(tmem, kTmemCols);
    else tmem_dealloc(tmem, kTmemCols);
  }
}

template <int BN, bool PAIR, int QKV, bool DS = false>
static cudaError_t launch_bn(const CUtensorMap& tmA, const CUtensorMap& tmB,
                             const CUtensorMap& tmO, const CUtensorMap& tmK,
                             const CUtensorMap& tmV, const GemmParams& p, int num_sms,
                             cudaStream_t s) {
  using C = GemmCfg<BN, PAIR>;
  static const cudaError_t attr = cudaFuncSetAttribute(
      gemm_kernel<BN, PAIR, QKV, DS>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
  if (attr != cudaSuccess) return attr;
  const int rows = PAIR ? 2 * kBM : kBM;
  const int tiles = ((p.M + rows - 1) / rows) * ((p.N + BN - 1) / BN);
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(192);
  cfg.dynamicSmemBytes = C::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  at[1].id = cudaLaunchAttributeClusterDimension;
  at[1].val.clusterDim.x = 2;
  at[1].val.clusterDim.y = 1;
  at[1].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = PAIR ? 2 : 1;
  int slots = num_sms;  // CTAs (pairs: CTA pairs) resident at once
  if (PAIR) {
    static int pairs = 0;  // CTA pairs that fit at once (one CTA per SM), asked once
    if (pairs == 0) {
      cfg.gridDim = dim3(2 * (num_sms / 2));
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, gemm_kernel<BN, PAIR, QKV>, &cfg) != cudaSuccess || n < 1) {
        cudaGetLastError();
        n = num_sms / 2;
      }
      pairs = n;
    }
    slots = pairs;
  }
  const int units = tiles < slots ? tiles : slots;
  cfg.gridDim = dim3(PAIR ? 2 * units : units);
  return cudaLaunchKernelEx(&cfg, gemm_kernel<BN, PAIR, QKV, DS>, tmA, tmB, tmO, tmK, tmV, p);
}

template <int QKV>
cudaError_t launch_gemm_t(const CUtensorMap& tmA, const CUtensorMap& tmB, const CUtensorMap& tmO,
                          const CUtensorMap& tmK, const CUtensorMap& tmV, const GemmParams& p,
                          int bn, bool pair, int num_sms, cudaStream_t s) {
  if (pair) {
    switch (bn) {
      case 96: return launch_bn<96, true, QKV>(tmA, tmB, tmO, tmK, tmV, p, num_sms, s);
      case 128: return launch_bn<128, true, QKV>(tmA, tmB, tmO, tmK, tmV, p, num_sms, s);
      case 192: return launch_bn<192, true, QKV>(tmA, tmB, tmO, tmK, tmV, p, num_sms, s);
      case 256: return launch_bn<256, true, QKV>(tmA, tmB, tmO, tmK, tmV, p, num_sms, s);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (bn) {
    case 64: return launch_bn<64, false, QKV>(tmA, tmB, tmO, tmK, tmV, p, num_sms, s);
    case 96: return launch_bn<96, false, QKV>(tmA, tmB, tmO, tmK, tmV, p, num_sms, s);
    case 128: return launch_bn<128, false, QKV>(tmA, tmB, tmO, tmK, tmV, p, num_sms, s);
    case 192: return launch_bn<192, false, QKV>(tmA, tmB, tmO, tmK, tmV, p, num_sms, s);
    case 256: return launch_bn<256, false, QKV>(tmA, tmB, tmO, tmK, tmV, p, num_sms, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace fd
