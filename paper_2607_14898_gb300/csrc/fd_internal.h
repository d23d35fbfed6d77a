// Internal launch interface between the host runtime (flashdec.cu) and the kernels
// (fd_gemm_kernel.cuh and its instances, fd_attn.cu, fd_small.cu). Not part of the public C ABI.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "flashdec.h"

namespace fd {

// Launch with programmatic stream serialization (the kernel must call grid_dep_wait before it
// touches memory written by the previous kernel of the stream).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

constexpr int kHeadDim = 64;     // D_h: every model size of the paper uses D / N = 64
constexpr int kRopePairs = 32;   // D_h / 2 rotation pairs: 12 temporal, 10 row, 10 column
constexpr int kBM = 128;         // GEMM / attention tile rows (one TMEM lane per row)
constexpr int kBK = 64;          // K elements per stage (one 128-byte swizzle atom)

enum EpiKind : int {
  EPI_F32 = 0,    // out_f32[r][c] = acc + bias
  EPI_RESID = 1,  // out_f32[r][c] += acc + bias (residual stream, in place)
  EPI_GELU = 2,   // out_bf16[r][c] = bf16(GELU(acc + bias))
  EPI_TUP = 3,    // temporal upsampling: column tau*D + d of row l -> out_f32[tau*L + l][d]
  EPI_QKV = 4,    // bias, KV-norm, 3D-RoPE; Q to q_out, K/V into the cache ring slot
  EPI_SWIGLU = 5, // gated SiLU: accumulator columns in blocks of 64 (32 gate, 32 up of the same
                  // hidden units); out_bf16[r][32j + i] = bf16(SiLU(g + bg) * (u + bu))
  EPI_GELU_F8 = 6,  // out_f8[r][c] = e4m3(GELU(acc * col_scale + bias) * out_scale)
  EPI_SWIGLU_F8 = 7,  // gated: out_f8[r][32j + i] = e4m3(SiLU(g) u out_scale) with g, u the
                      // (acc * col_scale + bias) of the interleaved gate / up columns
  EPI_PIXEL = 8,  // head layer 2 with the pixel shuffle: row tau L + l, column c rs^2 + dy rs + dx
                  // -> pixel [c][tau][gy rs + dy][gx rs + dx] (l = gy gw + gx), clamped to
                  // [-1, 1] as fp32 or as its uint8 code; frames past pix.frames are not written
};

// The scores-backward GEMM (attention training): rows r of S / dP are (head, query) rows of
// one query chunk, Pc rows per head (padding rows r % Pc % Lp >= L), columns keys (padding keys
// c % Lp >= L); dS bf16 [M][N]; dS^T, P^T bf16 [N][M].
struct DsEpi {
  const float* lse;    // [M] log-sum-exp of the row's scaled scores (natural log)
  const float* delta;  // [M] rowsum(dO o O)
  float scale;         // 1 / sqrt(D_h)
  int Pc, Lp, L;
  __nv_bfloat16 *dS, *dST, *PT;
};

// Output of EPI_PIXEL (the pixel head folded into the last product of the decoder).
struct PixelEpi {
  void* out;        // [C][frames][gh rs][gw rs], fp32 or uint8
  int u8;
  int frames;       // frames written (rows tau L + l with tau >= frames are dropped)
  int tokens;       // L: rows per frame
  int gh, gw, rs;   // token grid and the spatial upscale (rs % 4 == 0, 32 % rs == 0)
};

// One stream of a batched QKV launch: its cache ring, chunk counter and temporal RoPE table.
struct QkvStream {
  __nv_bfloat16* k_ring;     // [groups][ring_pitch][64]
  __half* vt_ring;           // [groups][64][ring_pitch]
  const int* step_dev;       // chunk index t of the stream
  const float2* rope_t;      // [frames_per_chunk][band_t] of the stream's chunk
};

// Rotary / cache parameters of the fused QKV epilogue.
struct QkvEpi {
  int qk_norm;  // 0: RMSNorm K (knorm_g) and V (vnorm_g); 1: Q (vnorm_g holds Q's gain) and K
  int heads, groups;
  const float* knorm_g;      // [64] KV-norm gain for K
  const float* vnorm_g;      // [64] KV-norm gain for V
  __nv_bfloat16* q_out;      // [M][heads * 64]
  __nv_bfloat16* k_ring;     // [groups][ring_pitch][64]
  __half* vt_ring;           // [groups][64][ring_pitch]   (V stored transposed, fp16)
  int ring_pitch;            // key rows per group (>= window * rows_per_chunk, multiple of 128)
  int tokens;                // L_frm
  int grid_w;                // token-grid width W'/p
  int frames_per_chunk;      // 1 (backbone) or r_t (refinement)
  int window;                // W_frm in chunks
  const int* step_dev;       // chunk index t on the device, or null to use step_host
  int step_host;
  float eps;
  int band_t, band_s;        // pairs in the temporal band and in each spatial band
  const float2* rope_t;      // [frames_per_chunk][band_t] (cos, sin) of this chunk's frames
  float inv_freq_s[kRopePairs];  // base^(-2i/d_band) of the row / column pairs (fp32)
  // batched launch (streams > 0): the rows stack `streams` independent streams, stream_rows rows
  // each (frames_per_chunk blocks of frame_rows >= tokens rows; rows past `tokens` in a block
  // are padding and append nothing); ring, counter and RoPE table come from stream[i], and K /
  // V are stored row by row (the single-stream fields above are unused)
  int streams, stream_rows, frame_rows;
  const QkvStream* stream;
};

// Output of the GEMM epilogue goes through TMA bulk stores with these tensor maps (all boxes
// are 32-row slabs, 128-byte swizzled unless noted):
//   EPI_F32 / EPI_RESID  tmO: fp32 [M][ld_out], box {32, 32} (RESID uses a bulk reduce-add)
//   EPI_GELU             tmO: bf16 [M][ld_out], box {64, 32}
//   EPI_TUP              tmO: fp32 3D {D, L, r_t}, box {32, 32, 1}
//   EPI_QKV              tmO: Q bf16 [M][heads*64], box {64, 32};
//                        tmK: K ring 4D {64, M, W, G} (row, slot, group strides), box {64,32,1,1};
//                        tmV: V^T ring 4D {M, W, 64, G}, box {32, 1, 64, 1}, no swizzle
//                        (used when v_tma; needs M % 8 == 0), else direct stores
struct GemmParams {
  int M, N, K;
  int epi;
  int v_tma;
  const float* bias;         // [N]
  float* out_f32;            // EPI_F32 / EPI_RESID / EPI_TUP
  int ld_out;                // row pitch of out_f32 / out_bf16 (elements)
  __nv_bfloat16* out_bf16;   // EPI_GELU
  int tup_tokens, tup_hidden;
  QkvEpi qkv;
  int* err;
  // FP8 operands: A and W are e4m3 (K-blocks of 128 elements, kind::f8f6f4 MMAs); the
  // accumulator is dequantised per output column by col_scale (s_A * s_W[n]) in the fp32 and
  // GELU_F8 epilogues. out_scale: multiplier before the e4m3 rounding of EPI_GELU_F8.
  int fp8;
  const float* col_scale;
  uint8_t* out_f8;
  float out_scale;
  // W is never written by a kernel of the stream (the decoder's weights): its first stages may
  // load before the dependency on the previous kernel is resolved
  int w_static;
  PixelEpi pix;  // EPI_PIXEL
  DsEpi ds;      // the scores-backward instance
};
// EPI_PIXEL is compiled into the single-CTA 256-wide instance only
inline bool gemm_pixel_epilogue_ok(int bn, bool pair, int rs) {
  return bn == 256 && !pair && rs % 4 == 0 && 32 % rs == 0;
}

// one stream of a batched attention launch (grid y = stream): its ring's K and V^T maps, its
// chunk counter and error word
struct AttnStream {
  CUtensorMap k, vt;
  const int* step_dev;
  int* err;
};

struct AttnParams {
  int Lq;                    // query rows
  int heads, groups;
  int ring_pitch;            // key rows per group in the ring
  int rows_per_chunk;        // keys appended per chunk
  int window;
  const int* step_dev;       // t on the device (keys = min(t+1, W) * rows_per_chunk) or null
  int n_keys_host;           // used when step_dev is null
  __nv_bfloat16* out;        // [Lq][heads * 64]
  int ld_out;
  float scale_log2;          // log2(e) / sqrt(D_h)
  int* err;
  int lq_pad;                // query rows per head in the packed row space (Lq rounded up to 8)
  int parts;                 // CTAs of the persistent launch; each takes an equal run of the
                             // (tile pair, key block) units
  float* part_o;             // [parts][2 slots][2 tiles][16][128 rows] float4 partial O
  float* part_ml;            // [parts][2][2][128] (running max, row sum)
  int* counters;             // [pairs] partial results stored per pair; zero between launches
  // batched launch over n_streams streams (null: one stream, the maps passed to the launch):
  // stream y's Q rows start at row y * q_rows_stream of tmQ, its output rows likewise in out,
  // its partial results and counters at y * ws_stride floats past part_o / part_ml / counters
  const AttnStream* streams;
  int n_streams;
  int q_rows_stream;
  size_t ws_stride;
  // batched only, optional: each row's natural-log log-sum-exp of the scaled scores, at
  // lse[(stream * heads + head) * lse_pitch + row] (the training step's backward)
  float* lse;
  int lse_pitch;
};

// launch wrappers; return cudaGetLastError() of the launch
// pair: 256-row tiles computed by CTA pairs (cta_group::2; bn 96 / 128 / 192 / 256): tmA
// boxes of 128 rows as for single CTAs, tmB boxes of bn / 2 rows (each CTA loads half of W)
cudaError_t launch_gemm(const CUtensorMap& tmA, const CUtensorMap& tmB, const CUtensorMap& tmO,
                        const CUtensorMap& tmK, const CUtensorMap& tmV, const GemmParams& p,
                        int bn, bool pair, int num_sms, cudaStream_t s);
// the scores-backward instance (DS): S = Q K^T (tmA, tmB) and dP = dO V^T (tmdO, tmV), K = 64
cudaError_t launch_gemm_scores_bwd(const CUtensorMap& tmA, const CUtensorMap& tmB,
                                   const CUtensorMap& tmdO, const CUtensorMap& tmV,
                                   const GemmParams& p, int num_sms, cudaStream_t s);
// the EPI_QKV instances (launch_gemm forwards to it for that epilogue)
cudaError_t launch_gemm_qkv(const CUtensorMap& tmA, const CUtensorMap& tmB,
                            const CUtensorMap& tmO, const CUtensorMap& tmK,
                            const CUtensorMap& tmV, const GemmParams& p, int bn, bool pair,
                            int num_sms, cudaStream_t s);
// Attention (+ the combine of key-range splits when p.splits > 1).
// tmQ: Q [Lq][heads * 64] bf16 in boxes of 64 x 128 rows; tmQ8: the same in boxes of 64 x 8.
cudaError_t launch_attention(const CUtensorMap& tmQ, const CUtensorMap& tmQ8,
                             const CUtensorMap& tmK,
                             const CUtensorMap& tmVt, const AttnParams& p, cudaStream_t s);
// GQA row packing: the query rows of the heads that share KV group g form one row space,
// head after head, each head's rows padded to a multiple of 8 (so a TMA box of 8 rows never
// holds two heads); 128-row tiles run over that space and a CTA takes two tiles of one group.
__host__ __device__ inline int attention_lq_pad(int Lq) { return (Lq + 7) / 8 * 8; }
__host__ __device__ inline int attention_tiles_per_group(int Lq, int heads, int groups) {
  return ((heads / groups) * attention_lq_pad(Lq) + 127) / 128;
}
// tile pairs (two 128-row tiles of one KV group) of an attention
inline int attention_units(int Lq, int heads, int groups) {
  return groups * ((attention_tiles_per_group(Lq, heads, groups) + 1) / 2);
}
// CTAs of an attention launch over `units` tile pairs with nblk key blocks each
int attention_parts(int units, int nblk, int num_sms);
// Workspace of an attention launch with `parts` CTAs: one int counter per tile pair (room for
// `pairs` pairs, at the start so that launches with other part counts find them in place),
// then partial O and (max, sum) for two slots of two tiles per CTA.
constexpr size_t kAttnPartFloats = 4 * (64 * 128 + 2 * 128);
inline size_t attention_counter_floats(int pairs) { return (static_cast<size_t>(pairs) + 3) / 4 * 4; }
inline size_t attention_workspace_floats(int parts, int pairs) {
  return parts <= 1 ? 0 : attention_counter_floats(pairs) + static_cast<size_t>(parts) * kAttnPartFloats;
}
inline void attention_workspace_split(float* ws, int parts, int pairs, AttnParams& a) {
  a.counters = reinterpret_cast<int*>(ws);
  a.part_o = ws ? ws + attention_counter_floats(pairs) : nullptr;
  a.part_ml = ws ? a.part_o + static_cast<size_t>(parts) * 4 * 64 * 128 : nullptr;
}
cudaError_t launch_unshuffle(const float* z, int C, int H, int W, int p, __nv_bfloat16* x0,
                             cudaStream_t s);
cudaError_t launch_rmsnorm(const float* h, const float* g, int M, int D, float eps,
                           __nv_bfloat16* u, cudaStream_t s);
// u[r][c] = e4m3(rmsnorm(h)[r][c] * oscale)  (FP8 MLP input)
cudaError_t launch_rmsnorm_e4m3(const float* h, const float* g, int M, int D, float eps,
                                uint8_t* u, float oscale, cudaStream_t s);
// frame_rows: F rows per refined frame (0 = gh gw, the tokens of a frame)
cudaError_t launch_pixel_head(const float* F, int frames, int gh, int gw, int C, int rs,
                              int out_u8, void* pix, cudaStream_t s, int frame_rows = 0);
cudaError_t launch_kv_append(const float* k, const float* v, int groups, int rows, int slot,
                             int ring_pitch, __nv_bfloat16* k_ring, __half* vt_ring,
                             cudaStream_t s);
cudaError_t launch_advance(int* step_dev, cudaStream_t s);
// failure-path check: a bounded wait that runs out after limit_ns and records ERR_WAIT_CHECK
cudaError_t launch_wait_check(int* err, unsigned long long limit_ns, cudaStream_t s);
// Temporal RoPE table of one chunk: for each block of `frames[k]` frames per chunk (k < nsets),
// entries [off_k + tau][i] = (cos, sin)((t * frames[k] + tau) * inv_freq[i]), i < band_t,
// computed in fp64 (t read from step_dev, or t_host when step_dev is null).
cudaError_t launch_rope_table(const int* step_dev, int t_host, int nsets, const int* frames,
                              int band_t, const double* inv_freq, float2* table,
                              cudaStream_t s);
constexpr int kMaxRopeSets = 2;

// ---- hooks of the training step (fd_train.cu) into the runtime (flashdec.cu)
// the weights object's configuration; device address of every blob tensor in blob order
// (returns the number of tensors); the weights object counts one more / one less user
const fd_config* weights_config(fd_weights w);
size_t weights_entries(fd_weights w, const void** ptrs, size_t n);
void weights_add_user(fd_weights w, int delta);
// out[M][N] (fp32, row pitch ldo) = A[M][K] (bf16, row pitch lda) W[N][K]^T (bf16, row pitch
// ldw) + bias, stored (EPI_F32) or added into out (EPI_RESID); pitches in elements, N % 32 == 0,
// lda, ldw % 8 == 0, ldo % 4 == 0, 16-byte aligned pointers
cudaError_t gemm_view(int epi, int M, int N, int K, const __nv_bfloat16* A, int lda,
                      const __nv_bfloat16* W, int ldw, const float* bias, float* out, int ldo,
                      int* err, cudaStream_t s);
// The attention's scores backward in one launch (the DS GEMM instance, 128 x 128 tiles):
// S = Q K^T and dP = dO V^T (Q, dO bf16 [M][64] with row pitch ldq; K, V bf16 [N][64] with row
// pitch ldk), then dS, dS^T, P^T as DsEpi describes. N % 32 == 0.
cudaError_t scores_bwd(int M, int N, const __nv_bfloat16* Q, const __nv_bfloat16* dO, int ldq,
                       const __nv_bfloat16* K, const __nv_bfloat16* V, int ldk, const DsEpi& ds,
                       int* err, cudaStream_t s);
// Band attention of the training step on the batched attention kernel, one "stream" per query
// chunk i: its keys are chunks max(0, i - W + 1) .. i of unpadded K bf16 [G][pitch][64] and
// V^T fp16 [G][64][pitch] (rows_per_chunk keys per chunk), so stream i's maps start at key
// max(0, i - W + 1) * rows_per_chunk and its key count is min(i + 1, W) rows_per_chunk with
// steps_dev[i] = i. Fills host[0 .. T-1]; false if a map cannot be made (the V^T start must
// be 16-byte aligned: rows_per_chunk % 8 == 0 unless T == 1).
bool band_attention_maps(AttnStream* host, int T, int W, int rows_per_chunk, int G, int pitch,
                         const __nv_bfloat16* k, const __half* vt, const int* steps_dev,
                         int* err);
// Q maps of the attention kernel over q bf16 [rows][heads 64]: boxes of 128 and of 8 rows
bool attention_q_maps(CUtensorMap* q, CUtensorMap* q8, const __nv_bfloat16* base, int rows,
                      int heads);

// GEMM tile widths compiled in
inline bool gemm_bn_supported(int bn) {
  return bn == 64 || bn == 96 || bn == 128 || bn == 192 || bn == 256;
}
// the QKV and GELU epilogues work on 64-column slabs (one head / one 128-byte bf16 row),
// the fp32 epilogues on 32-column slabs
inline bool gemm_bn_fits_epilogue(int bn, int epi) {
  if (epi == EPI_SWIGLU) return bn % 128 == 0;  // 128 accumulator columns -> 64 outputs
  if (epi == EPI_GELU_F8) return bn % 128 == 0;  // 128 e4m3 outputs per 128-byte slab row
  if (epi == EPI_SWIGLU_F8) return bn % 256 == 0;  // 256 accumulator columns -> 128 outputs
  return (epi == EPI_QKV || epi == EPI_GELU) ? bn % 64 == 0 : bn % 32 == 0;
}

}  // namespace fd
