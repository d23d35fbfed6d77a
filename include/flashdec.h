/*
 * flashdec.h - C ABI of the GB300 (sm_103a) FlashDecoder streaming decoder.
 *
 * The decoder turns one latent frame ("chunk") at a time into r_t pixel frames, keeping a
 * rolling key/value cache of the last W_frm chunks per attention layer (Sec. 3.3 "Streaming
 * with Rolling KV Cache", Eq. kv_cache, Algorithm 1). Per chunk t it runs:
 *   PixelUnshuffle(p) + Linear_{C' p^2 -> D}              (Eq. projection, Sec. 4.3)
 *   n_blocks x [RMSNorm, QKV + KV-norm + 3D-RoPE, attention over the cache, out-proj +
 *               residual, RMSNorm, MLP 4x (GELU) + residual]          (Sec. 3.2)
 *   RMSNorm, Linear_{D -> r_t D}, channel -> time reshape    (Eq. temporal_upsample)
 *   n_refine x the same block on r_t L tokens, window r_t W  (Sec. 3.4 "Step 2")
 *   RMSNorm, Linear_{D->D} + GELU, Linear_{D -> C r_s^2}, PixelShuffle(r_s), clamp
 *                                                             (Sec. 3.4 "Step 3")
 * Every step runs in the library's own CUDA kernels on the caller's stream.
 *
 * Conventions
 *   - All calls return fd_status; none throws, exits or traps.
 *   - Device pointers are CUDA device addresses on the current device; a stream argument is a
 *     cudaStream_t passed as void* (NULL = the legacy default stream).
 *   - A handle is not thread-safe; distinct handles may be used from distinct threads.
 *   - One GPU per process: the library caches the SM count, the kernels' shared-memory
 *     attributes and the cluster occupancy for the first device it runs on. Serve several GPUs
 *     with one process each (independent streams share nothing but the weights).
 *   - Asynchronous device errors (a kernel's bounded wait giving up, a CUDA launch error)
 *     put the handle in the FD_ERR_STATE state: later decode calls fail until fd_reset.
 */
#ifndef FLASHDEC_H
#define FLASHDEC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  FD_OK = 0,
  FD_ERR_INVALID_ARG = 1,     /* null / misaligned pointer, wrong size, bad enum          */
  FD_ERR_CONFIG = 2,          /* configuration outside what the kernels support           */
  FD_ERR_OOM = 3,             /* device allocation failed                                 */
  FD_ERR_CUDA = 4,            /* a CUDA runtime call or kernel launch failed              */
  FD_ERR_STATE = 5,           /* handle is in an error state: fd_reset it                 */
  FD_ERR_DEVICE_TIMEOUT = 6,  /* a kernel's bounded wait gave up (see fd_sync_status)     */
  FD_ERR_UNSUPPORTED = 7      /* device is not sm_103 / sm_100 class                      */
} fd_status;

typedef enum { FD_DTYPE_F32 = 0, FD_DTYPE_BF16 = 1, FD_DTYPE_U8 = 2 } fd_dtype;

/*
 * Decoder shape (names follow the paper: Sec. 3, Algorithm 1, Table "Model scaling").
 * Supported: hidden / heads == 64 (D_h), heads % kv_groups == 0, hidden % 128 == 0,
 * latent_h and latent_w divisible by patch, window >= 1, r_t >= 1, n_blocks >= 1,
 * out_channels * (vae_spatial * patch)^2 % 64 == 0.
 */
typedef struct {
  int32_t latent_channels; /* C'                                                  */
  int32_t latent_h;        /* H' (latent rows per frame)                          */
  int32_t latent_w;        /* W'                                                  */
  int32_t patch;           /* PixelUnshuffle factor p on the latent (Sec. 4.3)    */
  int32_t hidden;          /* D                                                   */
  int32_t heads;           /* N query heads                                       */
  int32_t kv_groups;       /* G key/value groups (GQA)                            */
  int32_t mlp_ratio;       /* MLP hidden = mlp_ratio * D                          */
  int32_t n_blocks;        /* backbone blocks                                     */
  int32_t n_refine;        /* temporal-refinement blocks                          */
  int32_t window;          /* W_frm, cached chunks including the current one      */
  int32_t r_t;             /* temporal upsampling factor (frames per chunk)       */
  int32_t vae_spatial;     /* pixels per latent cell side (8 for Wan2.1)          */
  int32_t out_channels;    /* C (3)                                               */
  int32_t out_dtype;       /* FD_DTYPE_F32 or FD_DTYPE_U8                         */
  int32_t mlp_gated;       /* MLP form: 0 = Linear, GELU, Linear; 1 = gated SiLU:    *
                            * SiLU(x Wg + bg) * (x Wu + bu), then Linear (XL layout) */
  float norm_eps;          /* RMSNorm epsilon (1e-6)                              */
  float rope_base;         /* RoPE base (10000)                                   */
  int32_t qk_norm;         /* per-head RMSNorm on: 0 = K and V (KV-norm, Sec. 3.2); *
                            * 1 = Q and K (QK-norm); the blob's second D_h gain is  *
                            * then Q's                                              */
  int32_t mlp_fp8;         /* 1: both products of every block MLP in FP8 (Sec. 4.6, *
                            * "static-calibrated FP8 quantization"): e4m3 weights   *
                            * with a power-of-two scale per row, e4m3 activations   *
                            * with static power-of-two scales derived from the      *
                            * weights at fd_weights_create (bounds that no input    *
                            * can exceed), fp32 accumulation. Needs mlp_gated = 0.  *
                            * The blob is unchanged.                                */
  int32_t first_chunk_frames; /* 0: every chunk emits r_t frames. 1: the causal frame *
                            * count of Fig. 2 (T' latent frames -> 1 + r_t (T'-1)   *
                            * frames): chunk 0 emits only its first refined frame   *
                            * (tau = 0; which one is kept is our reading), written  *
                            * as [C][1][H][W]; its cache entries are unchanged      */
  int32_t rope_mode;       /* temporal RoPE index: FD_ROPE_ABS or FD_ROPE_WINDOW_REL   */
} fd_config;

/*
 * Temporal index of the 3D-RoPE (Sec. 3.2), two readings of the paper:
 *   FD_ROPE_ABS         the offset t * L_frm of Algorithm 1: chunk t's frames sit at temporal
 *                       index t (backbone) and t r_t + tau (refinement); each key is rotated
 *                       once, when it enters the cache.
 *   FD_ROPE_WINDOW_REL  indices counted from the first frame of the current window (Sec. 4.3
 *                       "Long Video Decoding"), as if the whole window were re-rotated at
 *                       every chunk.
 * A score <R(a) q, R(b) k> depends only on b - a, and the window-relative indices of a query
 * and of a cached key differ by exactly what their absolute indices differ by, so the two
 * readings give the same scores. The library therefore runs one computation for both: keys
 * rotated once at their absolute index, with the temporal angles evaluated in double precision
 * for every chunk (so a long stream loses no accuracy to large indices). The mode is checked
 * and recorded; the pixels of the two modes are bit-identical.
 */
typedef enum { FD_ROPE_ABS = 0, FD_ROPE_WINDOW_REL = 1 } fd_rope_mode;

typedef struct fd_weights_s* fd_weights;
typedef struct fd_handle_s* fd_handle;
typedef struct fd_batch_s* fd_batch;

/* ------------------------------------------------------------------ sizes */

/* Number of elements of the weight blob for cfg (0 if cfg is invalid). Blob order, each
 * linear weight stored [out][in] row-major (nn.Linear layout):
 *   embed.w [D][C' p^2], embed.b [D]
 *   per backbone block b = 0 .. n_blocks-1:
 *     norm1.g [D], qkv.w [(N+2G)*64][D], qkv.b [(N+2G)*64], knorm.g [64], vnorm.g [64]
 *     (qnorm.g with qk_norm),
 *     out.w [D][N*64], out.b [D], norm2.g [D], mlp1.w [k*M*D][D], mlp1.b [k*M*D],
 *     mlp2.w [D][M*D], mlp2.b [D]
 *     (qkv rows: N query heads, then G key groups, then G value groups, 64 rows each;
 *      k = 1, or k = 2 with mlp_gated: the M*D gate rows, then the M*D up rows)
 *   normf.g [D], tup.w [r_t*D][D], tup.b [r_t*D]
 *   per refinement block: the same twelve tensors
 *   normh.g [D], head1.w [D][D], head1.b [D], head2.w [C r_s^2][D], head2.b [C r_s^2]
 * with r_s = vae_spatial * patch and M = mlp_ratio. */
size_t fd_weights_blob_elems(const fd_config* cfg);

/* Bytes of that blob for blob_dtype FD_DTYPE_F32 (4 per element) or FD_DTYPE_BF16 (2): the
 * blob_bytes fd_weights_create expects. 0 if cfg or blob_dtype is invalid. */
size_t fd_weights_blob_bytes(const fd_config* cfg, int blob_dtype);

/* Bytes of one latent chunk: C' * H' * W' fp32, layout [C'][H'][W'] row-major. */
size_t fd_latent_bytes(const fd_config* cfg);

/* Bytes of one chunk of pixels: C * r_t * (H' 8) * (W' 8) elements of out_dtype, layout
 * [C][r_t][H][W] row-major (planar channels, then frames; Sec. 3.4 Step 3). With
 * first_chunk_frames = 1, chunk 0 writes only the first 1/r_t of this ([C][1][H][W]). */
size_t fd_pixels_bytes(const fd_config* cfg);

/* Device bytes a handle allocates (rings, scratch), excluding the shared weights. */
size_t fd_handle_device_bytes(const fd_config* cfg);

/* ------------------------------------------------------------------ weights */

/* Load the parameters of the backbone B, the temporal refinement R and the projection / head
 * MLPs that Algorithm 1 takes as given ("Require: Backbone Transformer B, Temporal Refinement
 * Transformer R"; block layout Sec. 3.2, head Sec. 3.4 Step 3): copy a host weight blob
 * (order above) to the device, converting to bf16 (round to nearest even) for the linear
 * weights and keeping biases and gains in fp32.
 * blob_dtype: FD_DTYPE_F32 or FD_DTYPE_BF16. blob_bytes must equal
 * fd_weights_blob_bytes(cfg, blob_dtype). Synchronous. The caller keeps ownership of
 * host_blob; the library owns the device copy until fd_weights_destroy. A weights object may
 * be shared by several handles (it must outlive them).
 * Errors: FD_ERR_CONFIG (cfg invalid), FD_ERR_INVALID_ARG (null pointer, wrong size or
 * dtype), FD_ERR_OOM, FD_ERR_CUDA, FD_ERR_UNSUPPORTED; *out is set to NULL on error. */
fd_status fd_weights_create(const fd_config* cfg, const void* host_blob, size_t blob_bytes,
                            int blob_dtype, fd_weights* out);
/* Free a weights object. FD_ERR_STATE while a handle or batch still uses it. */
fd_status fd_weights_destroy(fd_weights w);

/* ------------------------------------------------------------------ streams */

/* Create a decoder stream state for cfg (must equal the weights' cfg): the initialisation
 * of Algorithm 1, (K^B, V^B) <- empty, (K^R, V^R) <- empty, t = 0. The caches are rings of the
 * sizes of Eq. kv_cache (Sec. 3.3): for every layer, backbone G x W L x 64 per K and V;
 * refinement G x r_t W L x 64; K bf16, V fp16 stored transposed. Also allocates the
 * activation scratch and the device chunk counter. Zero-fills the rings. Synchronous.
 * Errors: FD_ERR_CONFIG (cfg invalid or not the weights' cfg), FD_ERR_INVALID_ARG (null
 * pointer), FD_ERR_OOM, FD_ERR_CUDA, FD_ERR_UNSUPPORTED; *out is set to NULL on error. */
fd_status fd_create(const fd_config* cfg, fd_weights w, fd_handle* out);

/* Decode chunk t (Algorithm 1, one loop iteration) and advance t.
 * latent_dev: device fp32 [C'][H'][W'] (fd_latent_bytes), 16-byte aligned.
 * pixels_dev: device buffer of fd_pixels_bytes, 16-byte aligned, written with clamped
 *             pixels in [-1, 1] (fp32; NaN -> -1) or their uint8 codes
 *             q = round_half_even((clamp(x,-1,1) + 1) * 127.5) (uint8; NaN -> 0).
 * Both are used stream-ordered on `stream`; the call returns after enqueueing (no host
 * synchronisation). Attention at chunk t covers the min(t+1, W) most recent chunks. */
fd_status fd_decode_chunk(fd_handle h, const float* latent_dev, void* pixels_dev, void* stream);

/* Decode one chunk for each of n distinct handles (independent streams, e.g. sharing one
 * weights object). Ordered on `stream` as one operation: it starts after the work already on
 * `stream`, and work enqueued on `stream` afterwards sees every chunk's pixels. Inside, each
 * handle's chunk runs on a library-owned stream forked from and joined back to `stream`, so
 * the chunks run concurrently. All arguments are checked before anything is enqueued. */
fd_status fd_decode_chunks(fd_handle* hs, int n, const float* const* latents_dev,
                           void* const* pixels_dev, void* stream);

/* Batched decode (Sec. 4.6: independent streams share one set of weights). A batch object
 * owns stacked activation scratch for up to max_streams (1..64) streams of cfg: each stream's
 * L tokens are padded to Lp = 128 * ceil(L / 128) rows per frame, so every GEMM of a chunk
 * runs once on the rows of all streams, while attention and the pixel head run per stream on
 * that stream's own KV cache. The streams' states (KV rings, chunk counters) stay in their
 * fd_handles, created with the same weights object. Synchronous; counts as a user of w. */
fd_status fd_batch_create(const fd_config* cfg, fd_weights w, int max_streams, fd_batch* out);

/* Decode chunk t_i of each of n (1..max_streams) distinct handles through the batch object
 * and advance each t_i; the handles may be at different t. Pixels and latents as for
 * fd_decode_chunk (device, 16-byte aligned). Stream-ordered on `stream`, no host wait except
 * when the set of handles differs from the previous call (the batch's per-layer stream table
 * is then rewritten after a stream synchronisation). All arguments are checked before
 * anything is enqueued; a launch failure puts every handle of the call in the error state.
 * Calls with the same batch object must not overlap on different streams. */
fd_status fd_decode_batch(fd_batch b, fd_handle* hs, int n, const float* const* latents_dev,
                          void* const* pixels_dev, void* stream);

/* Free the batch object (after a device synchronisation). */
fd_status fd_batch_destroy(fd_batch b);

/* Like fd_decode_chunk, with the latent and the pixels in HOST memory (pinned for
 * asynchronous copies): the latent is copied into a library-owned device buffer, decoded, and
 * the pixels copied back, all stream-ordered on `stream`. The host buffers must stay valid
 * until the stream reaches the end of the copy-back. */
fd_status fd_decode_chunk_host(fd_handle h, const float* latent_host, void* pixels_host,
                               void* stream);

/* n consecutive chunks of the stream (Algorithm 1's loop, n times) from / to HOST memory, with
 * the copies overlapped with the decoding: while chunk t decodes on `stream`, chunk t+1's
 * latent is copied in and chunk t-1's pixels copied out on a library-owned copy stream (two
 * device buffers of each, used alternately). latents_host[t]: fp32 [C'][H'][W']
 * (fd_latent_bytes); pixels_host[t]: fd_pixels_bytes (a one-frame first chunk writes its first
 * 1/r_t). Pinned host memory for asynchronous copies. Stream-ordered: `stream` continues after
 * the last chunk's pixels are in host memory; the host buffers must stay valid until then. The
 * pixels are those of n fd_decode_chunk calls, bit for bit. The copy stream, events and the
 * second buffers are created on first use (2 * (latent + pixel) bytes of device memory at most).
 * Errors: FD_ERR_INVALID_ARG (null handle or pointer, n < 0), FD_ERR_STATE (handle in error,
 * or the chunk counter would pass 2^30), FD_ERR_OOM, FD_ERR_CUDA (the handle is then in error). */
fd_status fd_decode_sequence_host(fd_handle h, int n, const float* const* latents_host,
                                  void* const* pixels_host, void* stream);

/* Restart the stream: Algorithm 1's initialisation again for a new latent sequence, t = 0 and
 * the caches logically empty (their memory is not cleared; stale entries are never read
 * because attention at chunk t reads only chunks <= t). Clears the error state.
 * Stream-ordered: enqueued on the stream of the handle's last call, with no host wait. The
 * handle's next call that touches its device state (a decode, fd_load_state,
 * fd_debug_wait_timeout) is ordered after the reset whatever stream it is given: on another
 * stream it first waits for an event the reset recorded.
 * Errors: FD_ERR_INVALID_ARG (null handle), FD_ERR_CUDA. */
fd_status fd_reset(fd_handle h);

/* End of the stream (Algorithm 1 returns): free everything the handle owns, the caches
 * included, after synchronising its last stream. The handle is invalid afterwards; a batch
 * object that decoded it notices by the handle's serial number if the address comes back for
 * a new handle. Errors: FD_ERR_INVALID_ARG (null handle). */
fd_status fd_destroy(fd_handle h);

/* Host-side chunk counter (chunks decoded since create / reset). */
int64_t fd_chunk_index(fd_handle h);

/* Synchronise with the handle's last stream and read its device status word:
 * FD_OK, FD_ERR_DEVICE_TIMEOUT (a bounded wait gave up) or FD_ERR_CUDA. */
fd_status fd_sync_status(fd_handle h);

/* Static description of a status code. */
const char* fd_status_str(fd_status s);

/* Kernel kinds of the decode path, for the per-kernel profile. */
typedef enum {
  FD_K_UNSHUFFLE = 0, FD_K_EMBED = 1, FD_K_RMSNORM = 2, FD_K_QKV = 3, FD_K_ATTN_B = 4,
  FD_K_ATTN_R = 5, FD_K_OUT = 6, FD_K_MLP1 = 7, FD_K_MLP2 = 8, FD_K_TUP = 9, FD_K_HEAD1 = 10,
  FD_K_HEAD2 = 11, FD_K_PIXEL = 12, FD_K_ADVANCE = 13, FD_K_ROPE = 14, FD_K_COUNT = 15
} fd_kernel_kind;

/* Per-kernel profile (tracing): while enabled, every kernel the handle launches is bracketed
 * by CUDA events on its stream. fd_profile_collect synchronises, adds each kind's launch count
 * and device milliseconds into launches[FD_K_COUNT] / ms[FD_K_COUNT] (caller zeroes them) and
 * clears the recorded events. Attention is split into backbone (FD_K_ATTN_B) and refinement
 * (FD_K_ATTN_R) launches. */
fd_status fd_profile_enable(fd_handle h, int enable);
fd_status fd_profile_collect(fd_handle h, int64_t* launches, double* ms);

/* Number of kernels this handle has launched since fd_create. */
int64_t fd_launch_count(fd_handle h);

/* Streaming state, for checkpoint / resume and for moving a stream to another handle (no
 * counterpart in the paper, whose decode keeps this state in the process): the chunk index t
 * and every layer's rolling cache (backbone and refinement rings, K bf16 and V^T fp16, as the
 * device holds them). It contains no weights.
 *   fd_state_bytes: size of the state of a handle of configuration cfg (0 if cfg is invalid).
 *   fd_save_state: copy the handle's state into host_buf (exactly fd_state_bytes bytes), ordered
 *     on `stream` after the decodes already enqueued there (use the decode stream): the buffer
 *     is complete once the stream reaches this point. Pinned memory makes the copy asynchronous.
 *     FD_ERR_STATE if the handle is in error.
 *   fd_load_state: restore a saved state into a handle created with an identical configuration
 *     (checked against the header; FD_ERR_INVALID_ARG otherwise), ordered on `stream`; the next
 *     fd_decode_chunk on that stream continues the saved stream exactly as the original handle
 *     would have. Clears the handle's error state. */
size_t fd_state_bytes(const fd_config* cfg);
fd_status fd_save_state(fd_handle h, void* host_buf, size_t bytes, void* stream);
fd_status fd_load_state(fd_handle h, const void* host_buf, size_t bytes, void* stream);

/* Failure-path check (tests): enqueue on `stream` one kernel that waits, through the same
 * bounded mbarrier wait every decode kernel uses, on a barrier that nothing arrives at, with a
 * limit of limit_us microseconds (1 .. 100000) instead of the decode kernels' 2 s. The wait gives
 * up, records its code in the handle's device status word and the kernel returns (no trap, no
 * fault), exactly as a decode kernel does when a load or an MMA never completes. Afterwards
 * fd_sync_status returns FD_ERR_DEVICE_TIMEOUT, decode calls return FD_ERR_STATE, and fd_reset
 * makes the handle usable again. FD_ERR_INVALID_ARG for a null handle or a limit out of range. */
fd_status fd_debug_wait_timeout(fd_handle h, unsigned int limit_us, void* stream);

/* ------------------------------------------------------------------ training step */

/* One streaming training step (Sec. 3.3 "Training--Inference Consistency"; Sec. 3.5 Eq. loss,
 * its L1 term): the loss of a clip of T latent frames against its target video and the
 * gradient of every decoder parameter. Training through the rolling cache has the gradient of
 * one pass over the clip under the block sliding-window mask, and the step computes exactly
 * that: every chunk's forward with its activations kept (the attention of query chunk i over
 * key chunks i-W < j <= i), the L1 term, then the backward, all in the library's kernels (the
 * products on the tcgen05 GEMM, bf16 operands, fp32 accumulation).
 * Readings: the loss takes the head's output before the clamp (T1); the mean of |x_hat - x|
 * over every pixel of the clip (T3); the gradient flows through the cache (T2).
 *   fd_train_create: a trainer for clips of `chunks` (1 .. 256) latent frames of cfg (equal to
 *     the weights' cfg; the bf16-valued decoder with either MLP form and either first-chunk
 *     rule: mlp_fp8 gives FD_ERR_CONFIG). Allocates the saved activations and scratch,
 *     transposes the weights; synchronous. The trainer is a user of w.
 *   fd_train_step: latents device fp32 [T][C'][H'][W']; targets device fp32
 *     [T][C][r_t][H' 8][W' 8] (the pixels of each chunk, fd_pixels_bytes apart; with
 *     first_chunk_frames = 1, chunk 0's frames 1 .. r_t-1 are not read and the mean runs over
 *     the (T - 1) r_t + 1 frames the clip decodes to); loss: one
 *     device fp32; grads: device fp32 of fd_train_grad_elems(cfg) elements, written in the
 *     weight-blob order (each tensor's gradient where its weights sit in the blob). 16-byte
 *     aligned buffers. Enqueued on `stream`; a trainer runs one step at a time.
 *   fd_train_status: synchronise `stream`, then FD_OK, or FD_ERR_DEVICE_TIMEOUT if a kernel's
 *     bounded wait gave up during the last step.
 * Errors: FD_ERR_INVALID_ARG, FD_ERR_CONFIG, FD_ERR_OOM, FD_ERR_CUDA. */
typedef struct fd_trainer_s* fd_trainer;
size_t fd_train_grad_elems(const fd_config* cfg);
fd_status fd_train_create(const fd_config* cfg, fd_weights w, int chunks, fd_trainer* out);
fd_status fd_train_step(fd_trainer tr, const float* latents, const float* targets, float* loss,
                        float* grads, void* stream);
fd_status fd_train_status(fd_trainer tr, void* stream);
fd_status fd_train_destroy(fd_trainer tr);

/* Kernel kinds of the training step, for its per-kernel profile. */
enum fd_train_kind {
  FD_TK_LINEAR = 0,     /* forward products of the linears (embedding, blocks, upsampling, head) */
  FD_TK_DGRAD = 1,      /* their input gradients, dX = dY W */
  FD_TK_WGRAD = 2,      /* their weight gradients, dW = dY^T X */
  FD_TK_ATTN_GEMM = 3,  /* the attention's products: S = Q K^T (forward and recomputed), P V,
                           dP = dO V^T, dQ = dS K, dK = dS^T Q, dV = P^T dO */
  FD_TK_SOFTMAX = 4,    /* band softmax, row dot delta = rowsum(dO o O), softmax backward */
  FD_TK_TRANSPOSE = 5,  /* operand transposes for the products */
  FD_TK_NORM = 6,       /* RMSNorm forward / backward, KV-norm (QK-norm) + 3D-RoPE fwd / bwd */
  FD_TK_POINTWISE = 7,  /* bf16 casts, GELU forward / backward, copies, column sums, the
                           PixelUnshuffle, upsampling permutes and the L1 loss */
  FD_TK_COUNT = 8
};
/* Per-kernel profile of the training step: while enabled, every launch of fd_train_step is
 * bracketed by CUDA events on its stream. fd_train_profile_collect synchronises the device,
 * adds each kind's launch count and device milliseconds into launches[FD_TK_COUNT] /
 * ms[FD_TK_COUNT] (the caller zeroes them) and releases the recorded events.
 * Errors: FD_ERR_INVALID_ARG (null arguments), FD_ERR_CUDA. */
fd_status fd_train_profile_enable(fd_trainer tr, int enable);
fd_status fd_train_profile_collect(fd_trainer tr, int64_t* launches, double* ms);

/* Copy layer `layer` of the backbone (which = 0) or refinement (which = 1) ring into host
 * memory: K as [G][W * rows][64] bf16 bits, then V as [G][W * rows][64] fp16 bits (rows =
 * L backbone, r_t L refinement; row slot*rows + r holds token r of the chunk in ring slot
 * `slot` = chunk index mod W). dst_bytes must be >= 2 * G * W * rows * 64 * 2. Synchronous.
 * For tests of the cache indexing. */
fd_status fd_debug_read_ring(fd_handle h, int which, int layer, void* dst_host,
                             size_t dst_bytes);

#ifdef __cplusplus
}
#endif

#endif /* FLASHDEC_H */
