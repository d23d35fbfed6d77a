/*
 * flashdec_ops.h - kernel-level entry points of the FlashDecoder library.
 *
 * Each call enqueues one of the decoder's kernels on caller-owned device buffers and returns
 * after enqueueing (stream-ordered, no host synchronisation). They exist so each step of the
 * decode path (Algorithm 1) can be checked and timed on its own; fd_decode_chunk runs the
 * same kernels. All pointers are device pointers unless stated; `stream` is a cudaStream_t
 * as void*. `err_dev` is a device int32 the kernel ORs error bits into when one of its
 * bounded waits gives up (1 TMA load, 2 MMA commit, 4 accumulator release, 8 shared-memory
 * alignment); the caller zeroes it and reads it after synchronising. Argument errors are
 * reported synchronously as FD_ERR_INVALID_ARG; nothing is launched then.
 */
#ifndef FLASHDEC_OPS_H
#define FLASHDEC_OPS_H

#include "flashdec.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  FD_EPI_F32 = 0,   /* out fp32 [M][N]  = A W^T + b                                   */
  FD_EPI_RESID = 1, /* out fp32 [M][N] += A W^T + b          (residual, Sec. 3.2)      */
  FD_EPI_GELU = 2,  /* out bf16 [M][N]  = GELU_erf(A W^T + b) (MLP, R7; head, Sec. 3.4) */
  FD_EPI_TUP = 3,   /* out fp32 [(N / tup_hidden) M][tup_hidden]: column tau*D + d of row
                       l goes to row tau*M + l, column d (Eq. temporal_upsample)          */
  FD_EPI_SWIGLU = 4 /* out bf16 [M][N/2]: gated SiLU MLP (XL layout). W and bias rows come in
                       blocks of 64: rows 64j..64j+31 gate and 64j+32..64j+63 up of hidden
                       units 32j..32j+31; out[m][32j+i] = SiLU(g + bg) * (u + bu)          */
} fd_epilogue;

/* Linear layer on the tensor cores (tcgen05, bf16 in, fp32 accumulate).
 * A bf16 [M][K] row-major; W bf16 [N][K] row-major (nn.Linear); bias fp32 [N].
 * Requires N % 32 == 0 (N % 64 == 0 for FD_EPI_GELU, N % 128 == 0 for FD_EPI_SWIGLU),
 * K % 8 == 0, 16-byte aligned A / W / out / bias. bn = output tile width (64, 96, 128, 192
 * or 256; 96 only for the fp32 epilogues, 128 or 256 for FD_EPI_SWIGLU; 0 = library choice). */
fd_status fd_op_linear(int epilogue, int M, int N, int K, const void* A, const void* W,
                       const float* bias, void* out, int tup_hidden, int bn, int* err_dev,
                       void* stream);

/* The same with the launch shape chosen by the caller: bn as above (0 = library choice of
 * everything), pair = 1 for 128-row tiles on single CTAs, 2 for 256-row tiles on CTA pairs
 * (tcgen05 cta_group::2: each CTA of the pair holds its 128 rows of A and half of W's bn rows,
 * the even CTA issues the pair's MMAs; bn 96 / 128 / 192 / 256), 0 = library choice. Results
 * do not depend on the shape. fd_op_linear runs an explicit bn on single CTAs. */
fd_status fd_op_linear_tiled(int epilogue, int M, int N, int K, const void* A, const void* W,
                             const float* bias, void* out, int tup_hidden, int bn, int pair,
                             int* err_dev, void* stream);

/* Temporal 3D-RoPE table of chunk t (Sec. 3.2, reading of Algorithm 1's "RoPE offset"):
 * table[tau][i] = (cos, sin)((t * frames_per_chunk + tau) * rope_base^(-2i/24)) for the
 * frames_per_chunk frames of the chunk and the 12 temporal pairs (fp32 values of an fp64
 * evaluation). table: device float [frames_per_chunk][12][2]. */
fd_status fd_op_rope_table(int t, int frames_per_chunk, float rope_base, float* table,
                           void* stream);

/* Fused QKV projection of one attention block (Sec. 3.2, Sec. 3.3 step (2)):
 *   [Q | K | V] = A Wqkv^T + b   (Wqkv rows: heads*64 query, groups*64 key, groups*64 value)
 *   K, V <- RMSNorm over the 64 head dims with gains knorm_g / norm2_g (KV-norm), or with
 *           qk_norm = 1: Q, K <- RMSNorm with gains norm2_g / knorm_g (QK-norm), V as is
 *   Q, K <- 3D-RoPE at temporal index t*frames_per_chunk + row / tokens (cos / sin from
 *           rope_t, the fd_op_rope_table of chunk t), row and column of token (row % tokens)
 *           in a grid of width grid_w (rope_base; bands 24/20/20 dims)
 *   q_out bf16 [M][heads*64];  K -> k_ring bf16 [groups][ring_pitch][64] rows
 *   (t mod window)*M + row;  V -> vt_ring fp16 [groups][64][ring_pitch] (transposed), same
 *   key index.  M = frames_per_chunk * tokens; ring_pitch % 128 == 0, >= window * M;
 *   bqkv, q_out and the rings 16-byte aligned. */
fd_status fd_op_qkv(int M, int K, const void* A, const void* Wqkv, const float* bqkv,
                    const float* knorm_g, const float* norm2_g, int qk_norm, int heads, int groups,
                    int tokens, int grid_w, int frames_per_chunk, int window, int t, float eps,
                    float rope_base, const float* rope_t, void* q_out, void* k_ring,
                    void* vt_ring, int ring_pitch, int bn, int* err_dev, void* stream);

/* Attention of Lq queries over the first n_keys keys of a ring (Sec. 3.3, Eq. kv_cache):
 *   out[r][n*64 + d] = sum_j softmax_j(q_n . k_j / 8) v_j[d],  KV group g = n / (heads/groups)
 * q bf16 [Lq][heads*64]; k_ring bf16 [groups][ring_pitch][64]; vt_ring fp16
 * [groups][64][ring_pitch]; out bf16 [Lq][heads*64]. 1 <= n_keys <= ring_pitch,
 * ring_pitch % 128 == 0. Ring entries past n_keys must hold finite values.
 * parts: CTAs of the launch (0 = library choice, one per SM; 1..4096). The launch is
 * persistent: the query rows of the heads of each KV group are packed into 128-row tiles, the
 * (tile pair x 128-key block) units are cut into `parts` equal runs, one per CTA, and a tile
 * pair whose keys fall into several runs is finished by combining partial results. With
 * parts > 1, `workspace` is a caller-owned device buffer of fd_attention_workspace_bytes(...)
 * bytes (16-byte aligned) that the call overwrites (its counters are cleared on `stream` first);
 * calls sharing it must not overlap. The combine order is fixed: results do not depend on
 * which CTA finishes first. */
size_t fd_attention_workspace_bytes(int Lq, int heads, int groups, int n_keys, int parts);
fd_status fd_op_attention(int Lq, int heads, int groups, const void* q, const void* k_ring,
                          const void* vt_ring, int ring_pitch, int n_keys, void* out,
                          int parts, void* workspace, int* err_dev, void* stream);

/* Allocation-free variant of fd_op_attention. The paper has no counterpart: this is a library
 * convenience for callers that cannot call cudaMalloc, for example plug-ins that must stay
 * inside a device-memory budget handed to them by a host framework (which owns every
 * allocation), and real-time loops that cannot afford the device synchronisation an allocation
 * may cause. Such callers can pass their own inputs and outputs but have no way to provide the
 * partial-result workspace.
 * This call takes that workspace from one array in the library's static device memory,
 * FD_STATIC_ATTN_SCRATCH_BYTES (32 MiB) on every GPU that loads the library, held until the
 * process exits. It allocates nothing: no cudaMalloc, cudaFree or allocating library routine.
 *   - Arguments and results are those of fd_op_attention without `workspace`. parts = 0 lets
 *     the library choose (one CTA per SM: about 135 KB per SM). If
 *     fd_attention_workspace_bytes(..., parts) would exceed the static size, the call returns
 *     FD_ERR_INVALID_ARG and launches nothing (pass fewer parts; parts = 1 uses no workspace).
 *   - The 32 MiB are reserved on a device when the library's device code is loaded there,
 *     which with CUDA's lazy module loading may be this call's first use on that device.
 *   - The first call in a CUDA context (per device, and again after a device reset, which
 *     makes a new context) looks up the array's device address with that context current
 *     (cudaGetSymbolAddress); make that first call before any stream capture begins.
 *   - Every call shares the one array; it clears the array's counters on `stream` (a memset,
 *     not an allocation) and writes every other entry it later reads. Calls whose kernels
 *     overlap on the GPU (unordered streams) race on the array and may return wrong results. */
#define FD_STATIC_ATTN_SCRATCH_BYTES (32u << 20)
fd_status fd_op_attention_static(int Lq, int heads, int groups, const void* q,
                                 const void* k_ring, const void* vt_ring, int ring_pitch,
                                 int n_keys, void* out, int parts, int* err_dev, void* stream);

/* Rolling-cache append (Algorithm 1, cache update): fp32 k, v [groups][rows][64] rounded to
 * nearest even into ring slot s = t mod window: k_ring[g][s*rows + r][d] (bf16) and
 * vt_ring[g][d][s*rows + r] (fp16). The oldest chunk's slot is overwritten (eviction). */
fd_status fd_op_kv_append(const float* k, const float* v, int groups, int rows, int window,
                          int t, int ring_pitch, void* k_ring, void* vt_ring, void* stream);

/* u bf16 [M][D] = h / sqrt(mean(h^2) + eps) * g   (RMSNorm, Sec. 3.2); D % 128 == 0. */
fd_status fd_op_rmsnorm(const float* h, const float* g, int M, int D, float eps, void* u,
                        void* stream);

/* The same with e4m3 output (the input of an FP8 MLP, Sec. 4.6):
 * u e4m3 [M][D] = e4m3(h / sqrt(mean(h^2) + eps) * g * out_scale), round to nearest even,
 * saturating at +-448. */
fd_status fd_op_rmsnorm_e4m3(const float* h, const float* g, int M, int D, float eps,
                             float out_scale, void* u, void* stream);

/* FP8 linear layer (the MLP products of the FP8 option, Sec. 4.6): A e4m3 [M][K], W e4m3
 * [N][K] (nn.Linear layout), col_scale fp32 [N] (the dequantisation s_A * s_W[n]), bias fp32
 * [N]; acc = sum_k A[m][k] W[n][k], exact e4m3 products accumulated in fp32 (tcgen05
 * kind::f8f6f4):
 *   FD_EPI_F32    out fp32 [M][N]  = acc * col_scale + bias
 *   FD_EPI_RESID  out fp32 [M][N] += acc * col_scale + bias
 *   FD_EPI_GELU   out e4m3 [M][N]  = e4m3(GELU(acc * col_scale + bias) * out_scale)
 *   FD_EPI_SWIGLU out e4m3 [M][N/2] = e4m3(SiLU(g) u * out_scale), g / u = acc * col_scale +
 *                 bias of the gate / up rows, interleaved in blocks of 32 as for fd_op_linear
 *                 (the FP8 gated MLP layer 1); N % 256 == 0
 * K % 16 == 0, N % 32 == 0 (N % 128 == 0 for FD_EPI_GELU), 16-byte aligned A / W / out /
 * bias / col_scale.
 * bn = output tile width (96 / 128 / 192 / 256, 128 or 256 for FD_EPI_GELU; 0 = choice). */
fd_status fd_op_linear_e4m3(int epilogue, int M, int N, int K, const void* A, const void* W,
                            const float* col_scale, const float* bias, void* out,
                            float out_scale, int bn, int* err_dev, void* stream);

/* PixelUnshuffle(p) of a latent frame z fp32 [C][H][W] into tokens x0 bf16 [(H/p)(W/p)][C p^2]
 * (Sec. 4.3; raster token order of Eq. projection). */
fd_status fd_op_unshuffle(const float* z, int C, int H, int W, int p, void* x0, void* stream);

/* Pixel head (Sec. 3.4 Step 3): F fp32 [frames * gh * gw][C rs^2] -> pixels
 * [C][frames][gh rs][gw rs], pix = clamp(F[tau*L + y/rs*gw + x/rs][c rs^2 + (y%rs) rs + x%rs],
 * -1, 1), as fp32 or uint8 code round_half_even((pix + 1) * 127.5) (NaN -> 0). rs % 4 == 0. */
fd_status fd_op_pixel_head(const float* F, int frames, int grid_h, int grid_w, int channels,
                           int rs, int out_dtype, void* pixels, void* stream);

/* Head layer 2 with the pixel shuffle folded into the product's epilogue (Sec. 3.4 Step 3;
 * the decoder's last product, run this way by fd_decode_chunk): in one launch, the pixels that
 * fd_op_pixel_head gives from fd_op_linear's F = A W^T + b, bit for bit, without storing F.
 * A bf16 [M][K], the rows of frame tau's tokens at tau L .. tau L + L - 1 (L = grid_h grid_w);
 * W bf16 [channels rs^2][K]; bias fp32 [channels rs^2]. The first `frames` frames (frames L <=
 * M) are written: pixels [channels][frames][grid_h rs][grid_w rs], fp32 clamped to [-1, 1]
 * (out_dtype FD_DTYPE_F32) or uint8 codes (FD_DTYPE_U8). 128 x 256 tiles on single CTAs. rs % 4 == 0, 32 % rs == 0,
 * K % 8 == 0, (channels rs^2) % 32 == 0; 16-byte aligned A / W / bias / pixels.
 * Errors: FD_ERR_INVALID_ARG, FD_ERR_CUDA; err_dev as for fd_op_linear. */
fd_status fd_op_linear_pixel(int M, int K, const void* A, const void* W, const float* bias,
                             int frames, int grid_h, int grid_w, int channels, int rs,
                             int out_dtype, void* pixels, int* err_dev, void* stream);

/* ---- single kernels of the training step (fd_train_step), for per-kernel checks ---- */

/* The attention's scores backward in one launch (the training step's, Sec. 3.3 attention with
 * its softmax derivative): S = Q K^T and dP = dO V^T on the tensor cores (never stored), then
 *   P = exp(S / sqrt(64) - lse[r]), dS = P (dP - delta[r]) / sqrt(64)
 * with P = 0 on padding query rows (r mod Pc mod Lp >= L) and padding keys (c mod Lp >= L),
 * written as dS bf16 [M][N], dS^T and P^T bf16 [N][M]. Q, dO bf16 [M][64]; K, V bf16 [N][64];
 * lse, delta fp32 [M]. N % 32 == 0, Pc % Lp == 0, 0 < L <= Lp; 16-byte aligned.
 * Errors: FD_ERR_INVALID_ARG, FD_ERR_CUDA; err_dev as for fd_op_linear. */
fd_status fd_op_scores_bwd(int M, int N, const void* Q, const void* dO, const void* K,
                           const void* V, const float* lse, const float* delta, int Pc, int Lp,
                           int L, void* dS, void* dST, void* PT, int* err_dev, void* stream);

/* RMSNorm backward (the derivative of y = x r g, r = (mean(x^2) + eps)^(-1/2), Sec. 3.2):
 * dx = r (dy g) - x r^3 sum_j(dy_j g_j x_j) / D and dg = sum over rows of dy x r.
 * x, dy, dx fp32 [M][D]; g, dg fp32 [D]; work: fp32 [M][D] scratch of the caller. */
fd_status fd_op_rmsnorm_bwd(const float* x, const float* g, const float* dy, int M, int D,
                            float eps, float* dx, float* dg, float* work, void* stream);

/* GELU backward, exact form: dz = da (Phi(z) + z phi(z)); fp32 z, da, dz and a bf16 copy of dz
 * (the operand of the next products), n elements each. */
fd_status fd_op_gelu_bwd(const float* z, const float* da, int64_t n, float* dz, void* dz_bf16,
                         void* stream);

/* The L1 term of one chunk's pixels through the pixel shuffle (Sec. 3.4 Step 3, Sec. 3.5 Eq.
 * loss): F fp32 [frames grid_h grid_w][channels rs^2] (refined token tau L + l), target fp32
 * [channels][frames][grid_h rs][grid_w rs]; loss = mean |PixelShuffle(F) - target| (one fp32)
 * and dF = sign(F - target) / (pixel count) in F's layout. work: fp32 scratch of
 * ceil(frames L channels rs^2 / 256) elements. */
fd_status fd_op_l1_pixel_bwd(const float* F, const float* target, int frames, int grid_h,
                             int grid_w, int channels, int rs, float* dF, float* loss,
                             float* work, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* FLASHDEC_OPS_H */
