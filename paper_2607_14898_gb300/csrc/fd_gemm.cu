// tcgen05 / TMEM bf16 GEMM with fused epilogues: out = epilogue(A W^T + bias).
//
// A: bf16 [M][K] row-major (activations), W: bf16 [N][K] row-major (nn.Linear weight), both
// K-major, loaded by TMA with the 128-byte swizzle into a ring of shared-memory stages.
// One persistent CTA per SM walks 128 x BN output tiles. Warp roles:
//   warp 0 (one lane)  TMA producer: stages of 128x64 (A) and BNx64 (W)
//   warp 1 (one lane)  MMA issuer: 4 x tcgen05.mma (K = 16 each) per stage into a TMEM
//                      accumulator; two accumulators so the epilogue of tile i overlaps the
//                      MMAs of tile i+1
//   warps 2-5          epilogue: each thread owns one accumulator row (TMEM lane) and
//                      applies the fused epilogue while storing it
// Fused epilogues (the linear layers of Sec. 3.2 / 3.4 and Eq. projection / temporal_upsample):
//   EPI_F32    out = acc + b                    (patch-embed, head layer 2)
//   EPI_RESID  h  += acc + b                    (out-projection, MLP layer 2: residual)
//   EPI_GELU   out = bf16(GELU(acc + b))        (MLP layer 1, head layer 1)
//   EPI_TUP    channel block tau of token l -> refined token tau*L + l   (Eq. temporal_upsample)
//   EPI_QKV    bias; KV-norm (RMS over D_h) on K and V; 3D-RoPE on Q and K; Q to its buffer,
//              K and V (transposed) into ring slot t mod W of the layer's cache (Sec. 3.3)
#include "fd_internal.h"
#include "fd_ptx.cuh"

namespace fd {

template <int BN>
struct GemmCfg {
  static constexpr int kStages = BN >= 256 ? 4 : 6;
  static constexpr int kABytes = kBM * kBK * 2;  // 16 KB
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kTmemCols = 2 * BN <= 128 ? 128 : (2 * BN <= 256 ? 256 : 512);
  static constexpr int kBarOffset = kStages * kStageBytes;
  static constexpr int kSmem = kBarOffset + 256;
  static_assert(kSmem <= 227 * 1024, "shared memory");
};

__device__ __forceinline__ float gelu_erf(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}

// cos / sin of the 32 rotation pairs of one token (3D-RoPE, reading: temporal pairs first,
// then row, then column; angle = position * base^(-2i/d_band)), argument reduced in fp64.
__device__ __forceinline__ void rope_table(const QkvEpi& q, int f, int y, int x, float* c,
                                           float* s) {
#pragma unroll
  for (int i = 0; i < kRopePairs; ++i) {
    const int pos = i < q.band_t ? f : (i < q.band_t + q.band_s ? y : x);
    double a = static_cast<double>(pos) * q.inv_freq[i];
    a -= 6.283185307179586 * rint(a * 0.15915494309189535);
    sincosf(static_cast<float>(a), &s[i], &c[i]);
  }
}

template <int BN>
__global__ void __launch_bounds__(192, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ GemmParams p) {
  using C = GemmCfg<BN>;
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

  const int m_tiles = (p.M + kBM - 1) / kBM;
  const int n_tiles = (p.N + BN - 1) / BN;
  const int tiles = m_tiles * n_tiles;
  const int nk = (p.K + kBK - 1) / kBK;

  if (threadIdx.x == 0) {
    if (!aligned) atomicOr(p.err, ERR_SMEM_ALIGN);
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(bar_full + 8 * s, 1);
      mbar_init(bar_empty + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(bar_tfull + 8 * a, 1);
      mbar_init(bar_tempty + 8 * a, 128);
    }
    mbar_init(bar_done, 1);
    fence_barrier_init();
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (aligned && warp == 0 && lane == 0) {
    // ------------------------------------------------------------ TMA producer
    int it = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x) {
      const int m0 = (tile / n_tiles) * kBM;
      const int n0 = (tile % n_tiles) * BN;
      for (int kb = 0; kb < nk; ++kb, ++it) {
        const int s = it % C::kStages;
        const uint32_t ph = (it / C::kStages) & 1;
        if (!mbar_wait(bar_empty + 8 * s, ph ^ 1, p.err, ERR_WAIT_MMA)) { ok = false; break; }
        mbar_expect_tx(bar_full + 8 * s, C::kStageBytes);
        tma_load_2d(sA + s * C::kABytes, &tmA, bar_full + 8 * s, kb * kBK, m0);
        tma_load_2d(sB + s * C::kBBytes, &tmB, bar_full + 8 * s, kb * kBK, n0);
      }
    }
    // drain: the loads issued last must land before the CTA may exit
    for (int j = it - 1; j >= 0 && j >= it - C::kStages; --j)
      mbar_wait(bar_full + 8 * (j % C::kStages), (j / C::kStages) & 1, p.err, ERR_WAIT_TMA);
  } else if (aligned && warp == 1 && lane == 0) {
    // ------------------------------------------------------------ MMA issuer
    const uint32_t idesc = idesc_bf16_f32(kBM, BN);
    int it = 0, tc = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x, ++tc) {
      const int acc = tc & 1;
      if (!mbar_wait(bar_tempty + 8 * acc, ((tc >> 1) & 1) ^ 1, p.err, ERR_WAIT_EPI)) break;
      tc_fence_after();
      const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc * BN);
      for (int kb = 0; kb < nk; ++kb, ++it) {
        const int s = it % C::kStages;
        if (!mbar_wait(bar_full + 8 * s, (it / C::kStages) & 1, p.err, ERR_WAIT_TMA)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = sA + s * C::kABytes;
        const uint32_t b0 = sB + s * C::kBBytes;
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k)
          mma_bf16_ss(d_tmem, sdesc_k_sw128(a0 + 32 * k), sdesc_k_sw128(b0 + 32 * k), idesc,
                      (kb | k) != 0);
        mma_commit(bar_empty + 8 * s);  // stage s free once these MMAs have read it
      }
      if (ok) mma_commit(bar_tfull + 8 * acc);
    }
    mma_commit(bar_done);
    mbar_wait(bar_done, 0, p.err, ERR_WAIT_MMA);
  } else if (aligned && warp >= 2) {
    // ------------------------------------------------------------ epilogue
    const int quarter = warp & 3;  // TMEM lanes this warp may read
    const int rloc = quarter * 32 + lane;
    int t = 0;
    if (p.epi == EPI_QKV) t = p.qkv.step_dev ? *p.qkv.step_dev : p.qkv.step_host;
    int tc = 0;
    for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++tc) {
      const int acc = tc & 1;
      const bool got = mbar_wait(bar_tfull + 8 * acc, (tc >> 1) & 1, p.err, ERR_WAIT_MMA);
      if (!__all_sync(0xffffffffu, got)) break;  // leave together: TMEM loads are collective
      tc_fence_after();
      const int m0 = (tile / n_tiles) * kBM;
      const int n0 = (tile % n_tiles) * BN;
      const int row = m0 + rloc;
      const bool row_ok = row < p.M;
      const uint32_t tbase =
          tmem + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(acc * BN);

      if (p.epi == EPI_QKV) {
        const QkvEpi& q = p.qkv;
        float rc[kRopePairs], rsn[kRopePairs];
        const int rows_chunk = q.frames_per_chunk * q.tokens;  // = M
        const int slot = t % q.window;
        if (row_ok) {
          const int l = row % q.tokens;
          const int f = t * q.frames_per_chunk + row / q.tokens;
          rope_table(q, f, l / q.grid_w, l % q.grid_w, rc, rsn);
        }
#pragma unroll 1
        for (int c = 0; c < BN; c += 64) {
          uint32_t r0[32], r1[32];
          __syncwarp();  // tcgen05.ld is warp-collective: reconverge first
          tmem_ld_32x32b_x32(tbase + c, r0);
          tmem_ld_32x32b_x32(tbase + c + 32, r1);
          tmem_ld_wait();
          const int col = n0 + c;
          if (!row_ok || col >= p.N) continue;
          float v[64];
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            v[j] = __uint_as_float(r0[j]) + __ldg(p.bias + col + j);
            v[32 + j] = __uint_as_float(r1[j]) + __ldg(p.bias + col + 32 + j);
          }
          const int hidx = col / kHeadDim;
          const bool is_q = hidx < q.heads;
          const bool is_k = !is_q && hidx < q.heads + q.groups;
          if (!is_q) {  // KV-norm: RMS over the head dimension, learned gain
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
          }
          if (is_q) {
            uint4* dst = reinterpret_cast<uint4*>(q.q_out + static_cast<size_t>(row) *
                                                                (q.heads * kHeadDim) +
                                                  hidx * kHeadDim);
#pragma unroll
            for (int j = 0; j < 8; ++j)
              dst[j] = make_uint4(pack_bf16x2(v[8 * j], v[8 * j + 1]),
                                  pack_bf16x2(v[8 * j + 2], v[8 * j + 3]),
                                  pack_bf16x2(v[8 * j + 4], v[8 * j + 5]),
                                  pack_bf16x2(v[8 * j + 6], v[8 * j + 7]));
          } else if (is_k) {
            const int g = hidx - q.heads;
            const size_t krow = static_cast<size_t>(g) * q.ring_pitch + slot * rows_chunk + row;
            uint4* dst = reinterpret_cast<uint4*>(q.k_ring + krow * kHeadDim);
#pragma unroll
            for (int j = 0; j < 8; ++j)
              dst[j] = make_uint4(pack_bf16x2(v[8 * j], v[8 * j + 1]),
                                  pack_bf16x2(v[8 * j + 2], v[8 * j + 3]),
                                  pack_bf16x2(v[8 * j + 4], v[8 * j + 5]),
                                  pack_bf16x2(v[8 * j + 6], v[8 * j + 7]));
          } else {
            const int g = hidx - q.heads - q.groups;
            __nv_bfloat16* dst = q.vt_ring + static_cast<size_t>(g) * kHeadDim * q.ring_pitch +
                                 slot * rows_chunk + row;
#pragma unroll
            for (int j = 0; j < 64; ++j)
              dst[static_cast<size_t>(j) * q.ring_pitch] = __float2bfloat16_rn(v[j]);
          }
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint32_t r[32];
          __syncwarp();  // tcgen05.ld is warp-collective: reconverge first
          tmem_ld_32x32b_x32(tbase + c, r);
          tmem_ld_wait();
          const int col = n0 + c;
          if (!row_ok || col >= p.N) continue;
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]) + __ldg(p.bias + col + j);
          if (p.epi == EPI_GELU) {
            uint4* dst =
                reinterpret_cast<uint4*>(p.out_bf16 + static_cast<size_t>(row) * p.ld_out + col);
#pragma unroll
            for (int j = 0; j < 4; ++j)
              dst[j] = make_uint4(pack_bf16x2(gelu_erf(v[8 * j]), gelu_erf(v[8 * j + 1])),
                                  pack_bf16x2(gelu_erf(v[8 * j + 2]), gelu_erf(v[8 * j + 3])),
                                  pack_bf16x2(gelu_erf(v[8 * j + 4]), gelu_erf(v[8 * j + 5])),
                                  pack_bf16x2(gelu_erf(v[8 * j + 6]), gelu_erf(v[8 * j + 7])));
          } else {
            float* dst;
            if (p.epi == EPI_TUP) {
              const int tau = col / p.tup_hidden;
              dst = p.out_f32 + (static_cast<size_t>(tau) * p.tup_tokens + row) * p.tup_hidden +
                    (col - tau * p.tup_hidden);
            } else {
              dst = p.out_f32 + static_cast<size_t>(row) * p.ld_out + col;
            }
            float4* d4 = reinterpret_cast<float4*>(dst);
            if (p.epi == EPI_RESID) {
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                float4 o = d4[j];
                o.x += v[4 * j];
                o.y += v[4 * j + 1];
                o.z += v[4 * j + 2];
                o.w += v[4 * j + 3];
                d4[j] = o;
              }
            } else {
#pragma unroll
              for (int j = 0; j < 8; ++j)
                d4[j] = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
            }
          }
        }
      }
      __syncwarp();
      tc_fence_before();
      mbar_arrive(bar_tempty + 8 * acc);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

template <int BN>
static cudaError_t launch_bn(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmParams& p,
                             int num_sms, cudaStream_t s) {
  using C = GemmCfg<BN>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(gemm_kernel<BN>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const int tiles = ((p.M + kBM - 1) / kBM) * ((p.N + BN - 1) / BN);
  const int grid = tiles < num_sms ? tiles : num_sms;
  gemm_kernel<BN><<<grid, 192, C::kSmem, s>>>(tmA, tmB, p);
  return cudaGetLastError();
}

cudaError_t launch_gemm(const CUtensorMap& tmA, const CUtensorMap& tmB, const GemmParams& p,
                        int bn, int num_sms, cudaStream_t s) {
  switch (bn) {
    case 64: return launch_bn<64>(tmA, tmB, p, num_sms, s);
    case 128: return launch_bn<128>(tmA, tmB, p, num_sms, s);
    case 256: return launch_bn<256>(tmA, tmB, p, num_sms, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace fd
