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
// The launch is persistent: `parts` CTAs (one per SM) share the (tile pair, key block) units
// evenly; see WorkRange below.
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
//   warp 8        TMA: the two Q tiles of each segment into one of two buffers, K and V^T
//                 blocks of 128 keys into a 3-stage ring
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
constexpr int kVSub = 64 * 128;              // V^T sub-tile [64 dims][64 keys] fp16
constexpr int kVBytes = 2 * kVSub;           // V^T block of 128 keys
constexpr int kOffQ = 0;                     // two buffers of two Q tiles
constexpr int kOffK = 4 * kQBytes;
constexpr int kOffV = kOffK + kStages * kKBytes;
constexpr int kOffBar = kOffV + kStages * kVBytes;
constexpr int kSmem = kOffBar + 512;
constexpr int kThreads = 352;
constexpr int kTmemCols = 512;
constexpr uint32_t kColS = 0, kColP = 256, kColO = 384;  // + 128 X, + 64 X, + 64 X
constexpr float kRescaleLog2 = 8.0f;
// barrier indices
constexpr int kBarQFull = 0,                 // [buffer] Q tiles of a segment landed
              kBarQFree = kBarQFull + 2,     // [buffer] both tiles' S MMAs of the segment done
              kBarKvFull = kBarQFree + 2, kBarKvEmpty = kBarKvFull + kStages,
              kBarS = kBarKvEmpty + kStages,   // [tile] S_X(J) computed
              kBarSFree = kBarS + 2,           // [tile] S_X(J) read by the softmax
              kBarP = kBarSFree + 2,           // [tile] P_X(J) written
              kBarPv = kBarP + 2,              // [tile] P V of block J completed
              kBarOFree = kBarPv + 2,          // [tile] O_X of a segment read by the softmax
              kBarDone = kBarOFree + 2,        // [tile] every MMA of the tile's issuer completed
              kBarTurn = kBarDone + 2,  // [tile][quarter] the other tile's warp of this SMSP
                                        // has finished its exponentials: this tile's turn
              kBarPartDone = kBarTurn + 8,  // [slot] the 8 softmax warps wrote the partial
                                            // result of the CTA's first (0) / last (1) segment
              kBarDecided = kBarPartDone + 2,  // the TMA thread has counted both partials
              kNumBars = kBarDecided + 1;
static_assert(kNumBars * 8 + 8 <= 512, "barrier area");
static_assert(kSmem <= 227 * 1024, "shared memory");
// partial results of one (CTA, slot, tile): O as [16][128 rows] float4, then (m, l) per row
constexpr int kPartO = 64 * 128;
}  // namespace attn

// The work of one launch is the sequence of (tile pair, key block) units, pair-major: unit
// u = pair * nblk + kb. CTA c of `parts` processes units [c W / parts, (c+1) W / parts), so the
// SMs stay evenly loaded whatever the number of pairs; its range is a run of segments (one
// pair, consecutive key blocks). A pair covered by one CTA is finished there; a pair cut across
// CTAs leaves partial results (unnormalised O, running max, row sum) and the CTA that finishes
// the pair's last part combines them.
struct WorkRange {
  int W, parts;
  __device__ int start(int c) const {
    return static_cast<int>(static_cast<long long>(c) * W / parts);
  }
  // the CTA whose range holds unit u
  __device__ int cta_of(int u) const {
    return static_cast<int>((static_cast<long long>(u + 1) * parts - 1) / W);
  }
  // with fewer units than CTAs some ranges are empty
  __device__ bool empty(int c) const { return start(c + 1) == start(c); }
  // is pair p cut across CTAs?
  __device__ bool split(int p, int nblk) const { return cta_of(p * nblk) != cta_of(p * nblk + nblk - 1); }
};

// Only the first and the last segment of a CTA's range can hold part of a pair (every segment
// between them is a whole pair): partial-result slot 0 / 1.
struct PartialSlots {
  int pair[2];
  bool has[2];
  __device__ PartialSlots(const WorkRange& wr, int u0, int len, int nblk) {
    pair[0] = u0 / nblk;
    pair[1] = (u0 + len - 1) / nblk;
    has[0] = len > 0 && wr.split(pair[0], nblk);
    has[1] = len > 0 && pair[1] != pair[0] && wr.split(pair[1], nblk);
  }
};

// position in a CTA's unit sequence: block J of the CTA, unit (pair, kb), segment s
struct Cursor {
  int pair, kb, seg;
  bool first, last;  // first / last block of its segment
  __device__ void begin(int u0, int len, int nblk) {
    pair = u0 / nblk;
    kb = u0 - pair * nblk;
    seg = 0;
    first = true;
    last = kb == nblk - 1 || len == 1;
  }
  // next block; `left` = blocks after the new one within the CTA's range
  __device__ void next(int left, int nblk) {
    if (++kb == nblk) {
      kb = 0;
      ++pair;
    }
    first = kb == 0;
    if (first) ++seg;
    last = kb == nblk - 1 || left == 0;
  }
};

// kBatched: grid y = stream of p.streams (K / V maps, counter and error word from there; Q,
// output and workspace offset by the stream)
// kLse (batched only): also write each row's log-sum-exp of the scaled scores (natural log) to
// p.lse[(stream * heads + head) * p.lse_pitch + row], for a backward that recomputes P
template <bool kBatched, bool kLse = false>
__global__ void __launch_bounds__(attn::kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmQ8,
                const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const __grid_constant__ AttnParams p) {
  using namespace attn;
  // the stream's own pointers in a batched launch; the single-stream kernel reads p directly
  struct {
    const CUtensorMap *k, *v;
    int* err;
    const int* step;
    __nv_bfloat16* out;
    float *po, *pml;
    int* cnt;
    int q_row0;
  } bs{};
  if constexpr (kBatched) {
    const int y = blockIdx.y;
    const AttnStream* as = p.streams + y;
    bs.k = &as->k;
    bs.v = &as->vt;
    bs.err = as->err;
    bs.step = as->step_dev;
    bs.q_row0 = y * p.q_rows_stream;
    bs.out = p.out + static_cast<size_t>(bs.q_row0) * p.ld_out;
    bs.po = p.part_o + y * p.ws_stride;
    bs.pml = p.part_ml + y * p.ws_stride;
    bs.cnt = p.counters + y * p.ws_stride;
  }
  const CUtensorMap* const mK = kBatched ? bs.k : &tmK;
  const CUtensorMap* const mV = kBatched ? bs.v : &tmV;
#define ERR_WORD (kBatched ? bs.err : p.err)
#define STEP_DEV (kBatched ? bs.step : p.step_dev)
#define OUT_ROWS (kBatched ? bs.out : p.out)
#define PART_O (kBatched ? bs.po : p.part_o)
#define PART_ML (kBatched ? bs.pml : p.part_ml)
#define COUNTERS (kBatched ? bs.cnt : p.counters)
#define Q_ROW0 (kBatched ? bs.q_row0 : 0)
  extern __shared__ __align__(1024) uint8_t smem[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t base = smem_u32(smem);
  const bool aligned = (base & 1023u) == 0;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  const uint32_t bar0 = smem_u32(bars);
  auto bar = [&](int i) { return bar0 + 8u * static_cast<uint32_t>(i); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + kNumBars);
  volatile int* decision = reinterpret_cast<volatile int*>(bars + kNumBars) + 1;  // [2 slots]

  const int hpg = p.heads / p.groups;
  const int pairs_per_group = (attention_tiles_per_group(p.Lq, p.heads, p.groups) + 1) / 2;

  if (threadIdx.x == 0) {
    if (!aligned) atomicOr(ERR_WORD, ERR_SMEM_ALIGN);
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar(kBarQFull + b), 1);
      mbar_init(bar(kBarQFree + b), 2);  // both tiles' issuers
    }
    for (int st = 0; st < kStages; ++st) {
      mbar_init(bar(kBarKvFull + st), 1);
      mbar_init(bar(kBarKvEmpty + st), 2);  // both tiles' issuers release a stage
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(bar(kBarS + x), 1);
      mbar_init(bar(kBarSFree + x), 128);
      mbar_init(bar(kBarP + x), 128);
      mbar_init(bar(kBarPv + x), 1);
      mbar_init(bar(kBarOFree + x), 128);
      mbar_init(bar(kBarDone + x), 1);
    }
    for (int i = 0; i < 8; ++i) mbar_init(bar(kBarTurn + i), 1);
    mbar_init(bar(kBarPartDone), 8);
    mbar_init(bar(kBarPartDone + 1), 8);
    mbar_init(bar(kBarDecided), 1);
    fence_barrier_init();
  }
  grid_dep_wait();  // Q and the ring written by the previous kernels; TMEM freed by their CTAs
  int n_keys = p.n_keys_host;
  if (STEP_DEV != nullptr) {
    const int t = *STEP_DEV;
    n_keys = (t + 1 < p.window ? t + 1 : p.window) * p.rows_per_chunk;
  }
  const int nblk = (n_keys + 127) / 128;
  const WorkRange wr{p.groups * pairs_per_group * nblk, static_cast<int>(gridDim.x)};
  const int u0 = wr.start(blockIdx.x);
  const int len = wr.start(blockIdx.x + 1) - u0;  // blocks of this CTA (may be 0)
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
    if (lane == 0 && aligned && len > 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmQ8);
      prefetch_tmap(mK);
      prefetch_tmap(mV);
      // Count this CTA's partial results once the softmax warps have stored them. The stores
      // reach this thread through the barrier (CTA scope); the gpu-scope fence before the
      // counter update publishes them all (fences are cumulative). The CTA that stores a
      // pair's last part combines the pair. Slot 0 is polled between loads, so that a CTA
      // that finished its first segment early does not end up combining that pair too.
      const PartialSlots ps(wr, u0, len, nblk);
      bool counted[2] = {!ps.has[0], !ps.has[1]};
      decision[0] = decision[1] = 0;
      auto count_slot = [&](int sl) {
        counted[sl] = true;
        const int pr = ps.pair[sl];
        int owners = 0;  // CTAs holding a part of the pair
        for (int c = wr.cta_of(pr * nblk); c <= wr.cta_of(pr * nblk + nblk - 1); ++c)
          owners += wr.empty(c) ? 0 : 1;
        __threadfence();
        const int prev = atomicAdd(COUNTERS + pr, 1);
        if (prev == owners - 1) {
          COUNTERS[pr] = 0;  // every part has arrived: ready for the next launch
          __threadfence();
          decision[sl] = 1;
        }
      };
      Cursor cur;
      cur.begin(u0, len, nblk);
      int J = 0;
      bool ok = true;
      for (; J < len && ok; ++J) {
        if (!counted[0] && mbar_test_wait(bar(kBarPartDone), 0)) count_slot(0);
        const int g = cur.pair / pairs_per_group;
        if (cur.first) {
          // Q of the segment's pair into buffer seg & 1, once the segment two back has done
          // its S MMAs
          const int qb = cur.seg & 1;
          if (cur.seg >= 2 &&
              !mbar_wait(bar(kBarQFree + qb), ((cur.seg >> 1) - 1) & 1, ERR_WORD, ERR_WAIT_MMA)) {
            ok = false;
            break;
          }
          mbar_expect_tx(bar(kBarQFull + qb), 2 * kQBytes);
          // A tile inside one head's rows is one 128-row box (rows past Lq read the fill
          // value); a tile across two heads is loaded in boxes of 8 rows (one 1024-byte
          // swizzle atom each, same shared-memory layout). Rows past the group's last head
          // load head 0's first rows; their outputs are not written.
          for (int x = 0; x < 2; ++x) {
            const int rho0 = (2 * (cur.pair - g * pairs_per_group) + x) * kBM;
            const int hl0 = rho0 / p.lq_pad;
            const int hl1 = (rho0 + kBM - 1) / p.lq_pad;
            const uint32_t dst = base + kOffQ + (2 * qb + x) * kQBytes;
            const uint32_t qbar = bar(kBarQFull + qb);
            if (hl0 >= hpg) {
              tma_load_2d(dst, &tmQ, qbar, g * hpg * kHeadDim, Q_ROW0);
            } else if (hl1 == hl0 || hl1 >= hpg) {
              tma_load_2d(dst, &tmQ, qbar, (g * hpg + hl0) * kHeadDim,
                          Q_ROW0 + rho0 - hl0 * p.lq_pad);
            } else {
              for (int b = 0; b < kBM / 8; ++b) {
                const int rho = rho0 + 8 * b;
                int hl = rho / p.lq_pad;
                int r = rho - hl * p.lq_pad;
                if (hl >= hpg) hl = r = 0;
                tma_load_2d(dst + b * 1024, &tmQ8, qbar, (g * hpg + hl) * kHeadDim, Q_ROW0 + r);
              }
            }
          }
        }
        const int st = J % kStages;
        if (!mbar_wait(bar(kBarKvEmpty + st), ((J / kStages) & 1) ^ 1, ERR_WORD, ERR_WAIT_MMA)) {
          ok = false;
          break;
        }
        const uint32_t b = bar(kBarKvFull + st);
        mbar_expect_tx(b, kKBytes + kVBytes);
        tma_load_2d(base + kOffK + st * kKBytes, mK, b, 0, g * p.ring_pitch + cur.kb * 128);
        tma_load_2d(base + kOffV + st * kVBytes, mV, b, cur.kb * 128, g * kHeadDim);
        tma_load_2d(base + kOffV + st * kVBytes + kVSub, mV, b, cur.kb * 128 + 64,
                    g * kHeadDim);
        if (J + 1 < len) cur.next(len - J - 2, nblk);
      }
      // nothing may be in flight when the CTA exits: the last two Q loads, the last KV loads
      const int nseg = cur.seg + 1;
      for (int sg = nseg - 1; sg >= 0 && sg >= nseg - 2; --sg)
        mbar_wait(bar(kBarQFull + (sg & 1)), (sg >> 1) & 1, ERR_WORD, ERR_WAIT_TMA);
      for (int i = J - 1; i >= 0 && i >= J - kStages; --i)
        mbar_wait(bar(kBarKvFull + i % kStages), (i / kStages) & 1, ERR_WORD, ERR_WAIT_TMA);
      for (int sl = 0; sl < 2; ++sl)
        if (!counted[sl] && mbar_wait(bar(kBarPartDone + sl), 0, ERR_WORD, ERR_WAIT_EPI))
          count_slot(sl);
      mbar_arrive(bar(kBarDecided));
    }
  } else if (warp == 9 || warp == 10) {
    // ------------------------------------------------------------ MMA issue for tile x
    // One issuing thread per tile, so neither tile's MMAs wait behind the other's events;
    // tcgen05.commit tracks only the MMAs of the thread that issues it.
    const int x = warp - 9;
    if (lane == 0 && aligned && len > 0) {
      const uint32_t idesc_s = idesc_bf16_f32(128, 128);
      const uint32_t idesc_o = idesc_f16_f32(128, 64);  // P and V^T are fp16
      // descriptors of the stage bases; K steps of 16 elements add 32 B (2 in the encoded
      // address field) inside the 128-byte swizzle atom
      const uint64_t dq0 = sdesc_k_sw128(base + kOffQ + x * kQBytes);
      const uint64_t dk0 = sdesc_k_sw128(base + kOffK);
      const uint64_t dv0 = sdesc_k_sw128(base + kOffV);
      const uint32_t s_tmem = tmem + kColS + 128u * x;
      const uint32_t p_tmem = tmem + kColP + 64u * x;
      const uint32_t o_tmem = tmem + kColO + 64u * x;
      // S_X(J) = Q_X K_J^T; after the last block of a segment, release its Q buffer
      auto issue_s = [&](int J, const Cursor& c) -> bool {
        const int qb = c.seg & 1;
        if (c.first && !mbar_wait(bar(kBarQFull + qb), (c.seg >> 1) & 1, ERR_WORD, ERR_WAIT_TMA))
          return false;
        if (!mbar_wait(bar(kBarKvFull + J % kStages), (J / kStages) & 1, ERR_WORD, ERR_WAIT_TMA))
          return false;
        tc_fence_after();
        const uint64_t dq = dq0 + static_cast<uint64_t>((2 * qb * kQBytes) >> 4);
        const uint64_t dk = dk0 + static_cast<uint64_t>(((J % kStages) * kKBytes) >> 4);
        mma4_bf16_ss(s_tmem, dq, dk, idesc_s, 0u);
        mma_commit(bar(kBarS + x));
        if (c.last) mma_commit(bar(kBarQFree + qb));
        return true;
      };
      Cursor cur;
      cur.begin(u0, len, nblk);
      bool ok = issue_s(0, cur);
      for (int J = 0; J < len && ok; ++J) {
        const int st = J % kStages;
        const Cursor here = cur;
        // S of the next block as soon as the softmax has read S(J)
        if (J + 1 < len) {
          cur.next(len - J - 2, nblk);
          ok = mbar_wait(bar(kBarSFree + x), J & 1, ERR_WORD, ERR_WAIT_EPI) && issue_s(J + 1, cur);
          if (!ok) break;
        }
        // P V of this block once P(J) is written; the first block of a segment overwrites O,
        // so it also waits until the softmax has read the previous segment's O
        ok = mbar_wait(bar(kBarP + x), J & 1, ERR_WORD, ERR_WAIT_EPI);
        if (ok && here.first && here.seg > 0)
          ok = mbar_wait(bar(kBarOFree + x), (here.seg - 1) & 1, ERR_WORD, ERR_WAIT_EPI);
        tc_fence_after();
        if (!ok) break;
        const uint64_t dv = dv0 + static_cast<uint64_t>((st * kVBytes) >> 4);
        // keys 0-63 of the block (P columns 0-31, V^T sub-block 0), then keys 64-127
        mma4_bf16_ts(o_tmem, p_tmem, dv, idesc_o, here.first ? 0u : 1u);
        mma4_bf16_ts(o_tmem, p_tmem + 32u, dv + static_cast<uint64_t>(kVSub >> 4), idesc_o, 1u);
        mma_commit(bar(kBarPv + x));
        mma_commit(bar(kBarKvEmpty + st));  // one of the two arrivals that free the stage
      }
      mma_commit(bar(kBarDone + x));
      mbar_wait(bar(kBarDone + x), 0, ERR_WORD, ERR_WAIT_MMA);
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
    Cursor cur;
    cur.begin(u0, len, nblk);
    for (int J = 0; J < len && ok; ++J) {
      if (J > 0) cur.next(len - J - 1, nblk);
      if (cur.first) {
        m_used = -INFINITY;
        l_run = 0.f;
      }
      const bool got = mbar_wait(bar(kBarS + x), J & 1, ERR_WORD, ERR_WAIT_MMA);
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
      const int valid = n_keys - cur.kb * 128;
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
      // still be reading P_X(J-1): only the store of P(J) and the rescale of O wait for it.
      // Warp q of tile 0 and warp q of tile 1 share one SMSP; they take turns on the
      // exponentials (tile 0 block J, tile 1 block J, tile 0 block J+1, ...), so each one's S
      // load, P V wait and P store run while the other computes.
      if (x == 1 || J > 0) {
        const bool turn = mbar_wait(bar(kBarTurn + 4 * x + quarter), (x == 1 ? J : J - 1) & 1,
                                    ERR_WORD, ERR_WAIT_EPI);
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
      // P_X and O_X are free once the P V of the previous block has completed (for the
      // first block of a segment the previous segment's output already waited for it)
      if (!cur.first) {
        const bool pv = mbar_wait(bar(kBarPv + x), (J - 1) & 1, ERR_WORD, ERR_WAIT_MMA);
        if (!__all_sync(0xffffffffu, pv)) {
          ok = false;
          break;
        }
        tc_fence_after();
      }
      const bool resc = grow && !cur.first;
      if (resc) l_run *= ex2_approx(m_used - m_new);
      if (__any_sync(0xffffffffu, resc)) {
        const float f = resc ? ex2_approx(m_used - m_new) : 1.0f;
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
      if (!cur.last) continue;

      // -------------------------------------------------------- output of the segment
      const bool done = mbar_wait(bar(kBarPv + x), J & 1, ERR_WORD, ERR_WAIT_MMA);
      if (!__all_sync(0xffffffffu, done)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float o[64];
      {
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
      tc_fence_before();
      mbar_arrive(bar(kBarOFree + x));  // O_X may take the next segment's first P V
      const int g = cur.pair / pairs_per_group;
      const int rho = (2 * (cur.pair - g * pairs_per_group) + x) * kBM + row;
      const int hl = rho / p.lq_pad;
      const int r = rho - hl * p.lq_pad;
      const bool valid_row = hl < hpg && r < p.Lq;
      __nv_bfloat16* out_row =
          OUT_ROWS + static_cast<size_t>(r) * p.ld_out + (g * hpg + hl) * kHeadDim;
      const int c_lo = wr.cta_of(cur.pair * nblk);
      const int c_hi = wr.cta_of(cur.pair * nblk + nblk - 1);
      if (c_lo == c_hi) {  // the whole pair was done here
        if (valid_row) {
          if constexpr (kLse)
            p.lse[(static_cast<size_t>(blockIdx.y) * p.heads + g * hpg + hl) * p.lse_pitch + r] =
                (m_used + __log2f(l_run)) * 0.69314718055994531f;
          const float inv = 1.0f / l_run;
          uint4* dst = reinterpret_cast<uint4*>(out_row);
#pragma unroll
          for (int k = 0; k < 8; ++k)
            dst[k] = make_uint4(pack_bf16x2(o[8 * k] * inv, o[8 * k + 1] * inv),
                                pack_bf16x2(o[8 * k + 2] * inv, o[8 * k + 3] * inv),
                                pack_bf16x2(o[8 * k + 4] * inv, o[8 * k + 5] * inv),
                                pack_bf16x2(o[8 * k + 6] * inv, o[8 * k + 7] * inv));
        }
        continue;
      }
      // partial result into slot 0 (first segment of this CTA's range) or 1 (last one)
      const int slot = wr.start(blockIdx.x) >= cur.pair * nblk ? 0 : 1;
      {
        const size_t pb = (static_cast<size_t>(blockIdx.x) * 2 + slot) * 2 + x;
        float4* po = reinterpret_cast<float4*>(PART_O) + pb * (kPartO / 4) + row;
#pragma unroll
        for (int k = 0; k < 16; ++k)
          po[k * 128] = make_float4(o[4 * k], o[4 * k + 1], o[4 * k + 2], o[4 * k + 3]);
        reinterpret_cast<float2*>(PART_ML)[pb * 128 + row] = make_float2(m_used, l_run);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(kBarPartDone + slot));
    }
    // ------------------------------------------------------------ combine of cut pairs
    // after the CTA's last segment: for each partial result whose pair this CTA completed,
    // O = sum_c 2^(m_c - M) O_c / sum_c 2^(m_c - M) l_c over the CTAs c holding a part of it
    const PartialSlots ps(wr, u0, len, nblk);
    if (ok && (ps.has[0] || ps.has[1])) {
      const bool decided = mbar_wait(bar(kBarDecided), 0, ERR_WORD, ERR_WAIT_EPI);
      ok = __all_sync(0xffffffffu, decided);
      for (int sl = 0; sl < 2 && ok; ++sl) {
        if (!ps.has[sl] || !decision[sl]) continue;
        const int pr = ps.pair[sl];
        const int g = pr / pairs_per_group;
        const int rho = (2 * (pr - g * pairs_per_group) + x) * kBM + row;
        const int hl = rho / p.lq_pad;
        const int r = rho - hl * p.lq_pad;
        if (hl >= hpg || r >= p.Lq) continue;
        const int c_lo = wr.cta_of(pr * nblk);
        const int c_hi = wr.cta_of(pr * nblk + nblk - 1);
        float M = -INFINITY;
        for (int c = c_lo; c <= c_hi; ++c) {
          if (wr.empty(c)) continue;
          const size_t pb = (static_cast<size_t>(c) * 2 + (wr.start(c) >= pr * nblk ? 0 : 1)) * 2 + x;
          M = fmaxf(M, __ldcg(reinterpret_cast<const float2*>(PART_ML) + pb * 128 + row).x);
        }
        float acc[64];
#pragma unroll
        for (int d = 0; d < 64; ++d) acc[d] = 0.f;
        float l = 0.f;
        for (int c = c_lo; c <= c_hi; ++c) {
          if (wr.empty(c)) continue;
          const size_t pb = (static_cast<size_t>(c) * 2 + (wr.start(c) >= pr * nblk ? 0 : 1)) * 2 + x;
          const float2 ml = __ldcg(reinterpret_cast<const float2*>(PART_ML) + pb * 128 + row);
          const float w = ex2_approx(ml.x - M);
          l = fmaf(w, ml.y, l);
          const float4* po = reinterpret_cast<const float4*>(PART_O) + pb * (kPartO / 4) + row;
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const float4 v = __ldcg(po + k * 128);
            acc[4 * k] = fmaf(w, v.x, acc[4 * k]);
            acc[4 * k + 1] = fmaf(w, v.y, acc[4 * k + 1]);
            acc[4 * k + 2] = fmaf(w, v.z, acc[4 * k + 2]);
            acc[4 * k + 3] = fmaf(w, v.w, acc[4 * k + 3]);
          }
        }
        const float inv = 1.0f / l;
        if constexpr (kLse)
          p.lse[(static_cast<size_t>(blockIdx.y) * p.heads + g * hpg + hl) * p.lse_pitch + r] =
              (M + __log2f(l)) * 0.69314718055994531f;
        uint4* dst = reinterpret_cast<uint4*>(OUT_ROWS + static_cast<size_t>(r) * p.ld_out +
                                              (g * hpg + hl) * kHeadDim);
#pragma unroll
        for (int k = 0; k < 8; ++k)
          dst[k] = make_uint4(pack_bf16x2(acc[8 * k] * inv, acc[8 * k + 1] * inv),
                              pack_bf16x2(acc[8 * k + 2] * inv, acc[8 * k + 3] * inv),
                              pack_bf16x2(acc[8 * k + 4] * inv, acc[8 * k + 5] * inv),
                              pack_bf16x2(acc[8 * k + 6] * inv, acc[8 * k + 7] * inv));
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

#undef ERR_WORD
#undef STEP_DEV
#undef OUT_ROWS
#undef PART_O
#undef PART_ML
#undef COUNTERS
#undef Q_ROW0

int attention_parts(int units, int nblk, int num_sms) {
  const long long w = static_cast<long long>(units) * nblk;
  return static_cast<int>(w < num_sms ? (w > 0 ? w : 1) : num_sms);
}

cudaError_t launch_attention(const CUtensorMap& tmQ, const CUtensorMap& tmQ8,
                             const CUtensorMap& tmK,
                             const CUtensorMap& tmVt, const AttnParams& p, cudaStream_t s) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(attn_kernel<false>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, attn::kSmem);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(attn_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               attn::kSmem);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(attn_kernel<true, true>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, attn::kSmem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  if (p.streams != nullptr && p.lse != nullptr)
    return launch_pdl(attn_kernel<true, true>, dim3(p.parts, p.n_streams), dim3(attn::kThreads),
                      attn::kSmem, s, tmQ, tmQ8, tmK, tmVt, p);
  if (p.streams != nullptr)
    return launch_pdl(attn_kernel<true>, dim3(p.parts, p.n_streams), dim3(attn::kThreads),
                      attn::kSmem, s, tmQ, tmQ8, tmK, tmVt, p);
  return launch_pdl(attn_kernel<false>, dim3(p.parts), dim3(attn::kThreads), attn::kSmem, s, tmQ,
                    tmQ8, tmK, tmVt, p);
}

}  // namespace fd
