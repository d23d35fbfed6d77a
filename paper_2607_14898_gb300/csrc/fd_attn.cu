// Chunk-window flash attention on tcgen05 (Sec. 3.3 "Attention Pattern", Eq. kv_cache).
//
// Query tile of 128 rows x one head per CTA; keys are the first n_keys rows of the layer's
// ring (the min(t+1, W) cached chunks: ring slots 0..c-1 always hold exactly those chunks,
// and softmax does not depend on key order). No mask tensor: only the ragged last key block
// is cut at n_keys. GQA: head n reads KV group n / (N / G).
//
// Per key block of 128 (warps 0-3 = 128 threads, one query row / TMEM lane per thread):
//   S  = Q K^T          tcgen05.mma M=128 N=128 K=64, fp32 in TMEM columns [0, 128)
//   softmax             each thread loads its S row, online max / sum in fp32 (log2 domain),
//                       writes P = exp2(s - m) as bf16 into a 128-byte-swizzled smem tile
//   O_blk = P V         tcgen05.mma M=128 N=64 K=128 with B = V^T from the transposed V ring,
//                       fp32 in TMEM columns [128, 192); the thread folds it into its
//                       register accumulator o = o * alpha + O_blk
// K / V^T blocks are double-buffered TMA loads; S for block j+1 is issued right after P V for
// block j, so it overlaps the O_blk read-back. Two CTAs per SM overlap one CTA's MMAs with the
// other's softmax.
#include "fd_internal.h"
#include "fd_ptx.cuh"

namespace fd {

namespace attn {
constexpr int kQBytes = 128 * 128;       // Q tile [128][64] bf16
constexpr int kKBytes = 128 * 128;       // K block [128 keys][64] bf16
constexpr int kVBytes = 2 * 64 * 128;    // V^T block: 2 sub-tiles [64 dh][64 keys] bf16
constexpr int kPBytes = 2 * 128 * 128;   // P: 2 sub-tiles [128 rows][64 keys] bf16
constexpr int kOffQ = 0;
constexpr int kOffK = kOffQ + kQBytes;               // 2 stages
constexpr int kOffV = kOffK + 2 * kKBytes;           // 2 stages
constexpr int kOffP = kOffV + 2 * kVBytes;
constexpr int kOffBar = kOffP + kPBytes;
constexpr int kSmem = kOffBar + 128;
constexpr int kTmemCols = 256;
constexpr uint32_t kColO = 128;
}  // namespace attn

__global__ void __launch_bounds__(128, 2)
    attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const __grid_constant__ AttnParams p) {
  using namespace attn;
  extern __shared__ __align__(1024) uint8_t smem[];
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const uint32_t base = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  const uint32_t bar_q = smem_u32(bars + 0);
  const uint32_t bar_kv = smem_u32(bars + 1);  // [2]
  const uint32_t bar_s = smem_u32(bars + 3);
  const uint32_t bar_o = smem_u32(bars + 4);
  const uint32_t bar_done = smem_u32(bars + 5);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 6);
  const bool aligned = (base & 1023u) == 0;

  const int q0 = blockIdx.x * kBM;
  const int head = blockIdx.y;
  const int g = head / (p.heads / p.groups);
  int n_keys = p.n_keys_host;
  if (p.step_dev != nullptr) {
    const int t = *p.step_dev;
    n_keys = (t + 1 < p.window ? t + 1 : p.window) * p.rows_per_chunk;
  }
  const int nblk = (n_keys + 127) / 128;
  const int key_row0 = g * p.ring_pitch;

  if (tid == 0) {
    if (!aligned) atomicOr(p.err, ERR_SMEM_ALIGN);
    mbar_init(bar_q, 1);
    mbar_init(bar_kv, 1);
    mbar_init(bar_kv + 8, 1);
    mbar_init(bar_s, 1);
    mbar_init(bar_o, 1);
    mbar_init(bar_done, 1);
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tlane = static_cast<uint32_t>(warp * 32) << 16;
  const uint32_t idesc_s = idesc_bf16_f32(128, 128);
  const uint32_t idesc_o = idesc_bf16_f32(128, 64);

  int last_loaded[2] = {-1, -1};  // block index last loaded into each K/V stage (thread 0)
  int last_waited[2] = {-1, -1};
  auto load_kv = [&](int j, int st) {
    const uint32_t b = bar_kv + 8 * st;
    mbar_expect_tx(b, kKBytes + kVBytes);
    tma_load_2d(base + kOffK + st * kKBytes, &tmK, b, 0, key_row0 + j * 128);
    tma_load_2d(base + kOffV + st * kVBytes, &tmV, b, j * 128, g * kHeadDim);
    tma_load_2d(base + kOffV + st * kVBytes + kVBytes / 2, &tmV, b, j * 128 + 64, g * kHeadDim);
    last_loaded[st] = j;
  };
  auto issue_s = [&](int j) {  // S = Q K_j^T  (thread 0 only); always commits bar_s
    const int st = j & 1;
    const bool got = mbar_wait(bar_kv + 8 * st, (j >> 1) & 1, p.err, ERR_WAIT_TMA);
    if (got) last_waited[st] = j;
    tc_fence_after();
    if (got) {
#pragma unroll
      for (int k = 0; k < 4; ++k)
        mma_bf16_ss(tmem, sdesc_k_sw128(base + kOffQ + 32 * k),
                    sdesc_k_sw128(base + kOffK + st * kKBytes + 32 * k), idesc_s, k != 0);
    }
    mma_commit(bar_s);
  };

  bool issued_any = false;
  if (aligned && nblk > 0 && tid == 0) {
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    mbar_expect_tx(bar_q, kQBytes);
    tma_load_2d(base + kOffQ, &tmQ, bar_q, head * kHeadDim, q0);
    load_kv(0, 0);
    if (nblk > 1) load_kv(1, 1);
    mbar_wait(bar_q, 0, p.err, ERR_WAIT_TMA);
    issue_s(0);
    issued_any = true;
  }

  const float sl2 = p.scale_log2;
  float m_run = -INFINITY, l_run = 0.f;
  float o[64];
#pragma unroll
  for (int d = 0; d < 64; ++d) o[d] = 0.f;

  const int my_row = tid;  // row within the tile == TMEM lane
  uint8_t* sP = smem + kOffP;
  bool fail = !aligned;     // block-uniform when the loop is left
  for (int j = 0; j < nblk && aligned; ++j) {
    fail |= !mbar_wait(bar_s, j & 1, p.err, ERR_WAIT_MMA);
    tc_fence_after();
    uint32_t sr[4][32];
    __syncwarp();
#pragma unroll
    for (int c = 0; c < 4; ++c) tmem_ld_32x32b_x32(tmem + tlane + 32 * c, sr[c]);
    tmem_ld_wait();
    const int valid = n_keys - j * 128;  // >= 1
    float mx = -INFINITY;
#pragma unroll
    for (int c = 0; c < 4; ++c)
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        float s = __uint_as_float(sr[c][e]);
        if (32 * c + e >= valid) s = -INFINITY;
        sr[c][e] = __float_as_uint(s);
        mx = fmaxf(mx, s);
      }
    const float m_new = fmaxf(m_run, mx * sl2);
    const float alpha = ex2_approx(m_run - m_new);
    float lsum = 0.f;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
#pragma unroll
      for (int e8 = 0; e8 < 4; ++e8) {
        float pv[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          pv[e] = ex2_approx(fmaf(__uint_as_float(sr[c][8 * e8 + e]), sl2, -m_new));
          lsum += pv[e];
        }
        const uint32_t key = 32 * c + 8 * e8;  // first key of this 16-byte chunk
        const uint32_t off = (key >> 6) * (128 * 128) + sw128_offset(my_row, key & 63);
        *reinterpret_cast<uint4*>(sP + off) =
            make_uint4(pack_bf16x2(pv[0], pv[1]), pack_bf16x2(pv[2], pv[3]),
                       pack_bf16x2(pv[4], pv[5]), pack_bf16x2(pv[6], pv[7]));
      }
    }
    l_run = l_run * alpha + lsum;
    m_run = m_new;
    fence_proxy_async_smem();  // P (generic-proxy stores) visible to the tensor core
    tc_fence_before();
    if (__syncthreads_or(fail)) {  // also orders every S / O_blk TMEM read before the MMAs
      fail = true;
      break;
    }
    if (tid == 0) {
      tc_fence_after();
      const uint32_t vst = base + kOffV + (j & 1) * kVBytes;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t sub = kk >> 2, within = (kk & 3) * 32;
        mma_bf16_ss(tmem + kColO, sdesc_k_sw128(base + kOffP + sub * (128 * 128) + within),
                    sdesc_k_sw128(vst + sub * (64 * 128) + within), idesc_o, kk != 0);
      }
      mma_commit(bar_o);
      if (j + 1 < nblk) issue_s(j + 1);
    }
    const bool o_ok = mbar_wait(bar_o, j & 1, p.err, ERR_WAIT_MMA);
    fail |= !o_ok;
    tc_fence_after();
    uint32_t orr[2][32];
    __syncwarp();
    tmem_ld_32x32b_x32(tmem + tlane + kColO, orr[0]);
    tmem_ld_32x32b_x32(tmem + tlane + kColO + 32, orr[1]);
    tmem_ld_wait();
#pragma unroll
    for (int d = 0; d < 32; ++d) {
      o[d] = fmaf(o[d], alpha, __uint_as_float(orr[0][d]));
      o[32 + d] = fmaf(o[32 + d], alpha, __uint_as_float(orr[1][d]));
    }
    tc_fence_before();
    if (tid == 0 && o_ok && j + 2 < nblk) load_kv(j + 2, j & 1);  // stage free: P V_j done
  }
  const bool ok = !fail;

  // output row: O / l as bf16
  const int row = q0 + my_row;
  if (ok && row < p.Lq) {
    const float inv = 1.0f / l_run;
    uint4* dst = reinterpret_cast<uint4*>(p.out + static_cast<size_t>(row) * p.ld_out +
                                          head * kHeadDim);
#pragma unroll
    for (int j = 0; j < 8; ++j)
      dst[j] = make_uint4(pack_bf16x2(o[8 * j] * inv, o[8 * j + 1] * inv),
                          pack_bf16x2(o[8 * j + 2] * inv, o[8 * j + 3] * inv),
                          pack_bf16x2(o[8 * j + 4] * inv, o[8 * j + 5] * inv),
                          pack_bf16x2(o[8 * j + 6] * inv, o[8 * j + 7] * inv));
  }

  // teardown: every MMA of this CTA has completed and no TMA load is still in flight
  if (tid == 0 && issued_any) {
    mma_commit(bar_done);
    mbar_wait(bar_done, 0, p.err, ERR_WAIT_MMA);
    for (int st = 0; st < 2; ++st)
      if (last_loaded[st] > last_waited[st])
        mbar_wait(bar_kv + 8 * st, (last_loaded[st] >> 1) & 1, p.err, ERR_WAIT_TMA);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

cudaError_t launch_attention(const CUtensorMap& tmQ, const CUtensorMap& tmK,
                             const CUtensorMap& tmVt, const AttnParams& p, cudaStream_t s) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         attn::kSmem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  dim3 grid((p.Lq + kBM - 1) / kBM, p.heads);
  attn_kernel<<<grid, 128, attn::kSmem, s>>>(tmQ, tmK, tmVt, p);
  return cudaGetLastError();
}

}  // namespace fd
