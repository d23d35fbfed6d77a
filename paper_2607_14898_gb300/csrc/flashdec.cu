// Host runtime of the C ABI (include/flashdec.h, include/flashdec_ops.h): configuration
// checks, device weights, per-stream state (KV rings, scratch, chunk counter), TMA
// descriptors, and the per-chunk kernel sequence of Algorithm 1.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp8.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <vector>

#include "fd_internal.h"
#include "flashdec.h"
#include "flashdec_ops.h"

using fd::kHeadDim;

namespace {

// ---------------------------------------------------------------- driver entry points
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool load_encode() {
  std::call_once(g_encode_once, [] {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return g_encode != nullptr;
}

// 2D bf16 tensor [outer][inner] with row pitch row_bytes, 128-byte swizzled box
// {box_inner (<= 64), box_outer}.
bool tmap_16bit(CUtensorMap* m, CUtensorMapDataType dt, const void* base, uint64_t inner,
                uint64_t outer, uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer) {
  if (!load_encode()) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return g_encode(m, dt, 2, const_cast<void*>(base), dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
bool tmap_bf16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
               uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer) {
  return tmap_16bit(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, base, inner, outer, row_bytes,
                    box_inner, box_outer);
}
bool tmap_f16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
              uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer) {
  return tmap_16bit(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, base, inner, outer, row_bytes,
                    box_inner, box_outer);
}

// N-d tensor map (rank <= 5): dims innermost first, strides in bytes for dims 1..rank-1
bool tmap_nd(CUtensorMap* m, CUtensorMapDataType dt, int rank, const void* base,
             const uint64_t* dims, const uint64_t* strides, const uint32_t* box,
             CUtensorMapSwizzle sw) {
  if (!load_encode()) return false;
  cuuint64_t d[5], st[4];
  cuuint32_t b[5], es[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    b[i] = box[i];
    es[i] = 1;
    if (i > 0) st[i - 1] = strides[i - 1];
  }
  return g_encode(m, dt, rank, const_cast<void*>(base), d, st, b, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// e4m3 K-major operand [outer][inner] bytes in boxes of 128 bytes x box_outer rows
bool tmap_e4m3(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
               uint64_t row_bytes, uint32_t box_outer) {
  const uint64_t dims[2] = {inner, outer}, strides[1] = {row_bytes};
  const uint32_t box[2] = {128, box_outer};
  return tmap_nd(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, base, dims, strides, box,
                 CU_TENSOR_MAP_SWIZZLE_128B);
}

// GEMM epilogue store maps (32-row slabs)
bool tmap_out_e4m3(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint64_t ld) {
  const uint64_t dims[2] = {cols, rows}, strides[1] = {ld};
  const uint32_t box[2] = {128, 32};
  return tmap_nd(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, base, dims, strides, box,
                 CU_TENSOR_MAP_SWIZZLE_128B);
}
bool tmap_out_f32(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint64_t ld) {
  const uint64_t dims[2] = {cols, rows}, strides[1] = {ld * 4};
  const uint32_t box[2] = {32, 32};
  return tmap_nd(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box,
                 CU_TENSOR_MAP_SWIZZLE_128B);
}
bool tmap_out_bf16(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint64_t ld) {
  const uint64_t dims[2] = {cols, rows}, strides[1] = {ld * 2};
  const uint32_t box[2] = {64, 32};
  return tmap_nd(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box,
                 CU_TENSOR_MAP_SWIZZLE_128B);
}
// temporal upsampling output viewed as [streams][r_t][L][D] (L rows per refined frame)
bool tmap_out_tup(CUtensorMap* m, const void* base, uint64_t D, uint64_t L, uint64_t rt,
                  uint64_t streams = 1) {
  const uint64_t dims[4] = {D, L, rt, streams};
  const uint64_t strides[3] = {D * 4, L * D * 4, rt * L * D * 4};
  const uint32_t box[4] = {32, 32, 1, 1};
  return tmap_nd(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, base, dims, strides, box,
                 CU_TENSOR_MAP_SWIZZLE_128B);
}
// K ring [G][pitch][64] viewed as {64, M rows of a slot, W slots, G}
bool tmap_kring_store(CUtensorMap* m, const void* base, uint64_t M, uint64_t W, uint64_t G,
                      uint64_t pitch) {
  const uint64_t dims[4] = {64, M, W, G};
  const uint64_t strides[3] = {128, M * 128, pitch * 128};
  const uint32_t box[4] = {64, 32, 1, 1};
  return tmap_nd(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, base, dims, strides, box,
                 CU_TENSOR_MAP_SWIZZLE_128B);
}
// V^T ring [G][64][pitch] (fp16) viewed as {M keys of a slot, W slots, 64 dims, G};
// needs M % 8 == 0
bool tmap_vring_store(CUtensorMap* m, const void* base, uint64_t M, uint64_t W, uint64_t G,
                      uint64_t pitch) {
  const uint64_t dims[4] = {M, W, 64, G};
  const uint64_t strides[3] = {M * 2, pitch * 2, 64 * pitch * 2};
  const uint32_t box[4] = {32, 1, 64, 1};
  return tmap_nd(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, base, dims, strides, box,
                 CU_TENSOR_MAP_SWIZZLE_NONE);
}

int g_num_sms = 0;
int num_sms() {
  if (g_num_sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (g_num_sms <= 0) g_num_sms = 1;
  }
  return g_num_sms;
}

fd_status check_device() {
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return FD_ERR_CUDA;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
    return FD_ERR_CUDA;
  if (major != 10 || minor != 3) return FD_ERR_UNSUPPORTED;  // built for sm_103a only
  return FD_OK;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ---------------------------------------------------------------- configuration
struct Dims {
  int C, H, W, p, D, N, G, Dh, Mr, nb, nr, Wn, rt, rs, Cout, cin, gh, gw, L, head_out, qkv_out;
  bool u8;
  bool gated;  // gated-SiLU MLP: layer 1 has 2 Mr D outputs (gate, up)
  bool qk;     // QK-norm instead of KV-norm
  bool fp8;    // block MLPs in FP8 (e4m3 operands, static scales)
  bool f1;     // chunk 0 emits one frame (first_chunk_frames = 1)
};

bool valid_cfg(const fd_config* c) {
  if (c == nullptr) return false;
  // upper bounds first, so that the int products below (heads x 64, C' p^2, C r_s^2, ...)
  // cannot overflow; every real decoder sits far inside them
  if (c->latent_channels > 4096 || c->patch > 16 || c->heads > 256 || c->kv_groups > 256 ||
      c->mlp_ratio > 16 || c->n_blocks > 1024 || c->n_refine > 1024 || c->window > 4096 ||
      c->r_t > 64 || c->vae_spatial > 64 || c->out_channels > 64 || c->latent_h > (1 << 16) ||
      c->latent_w > (1 << 16))
    return false;
  if (c->latent_channels < 1 || c->latent_h < 1 || c->latent_w < 1 || c->patch < 1) return false;
  if (c->latent_h % c->patch || c->latent_w % c->patch) return false;
  if (c->heads < 1 || c->kv_groups < 1 || c->heads % c->kv_groups) return false;
  if (c->hidden != c->heads * kHeadDim || c->hidden % 128) return false;
  if (c->mlp_ratio < 1 || c->n_blocks < 1 || c->n_refine < 0 || c->window < 1 || c->r_t < 1)
    return false;
  if (c->vae_spatial < 1 || c->out_channels < 1) return false;
  const int rs = c->vae_spatial * c->patch;
  if (rs % 4) return false;
  if ((c->out_channels * rs * rs) % 64) return false;
  if ((c->latent_channels * c->patch * c->patch) % 8) return false;  // TMA row pitch
  if (c->out_dtype != FD_DTYPE_F32 && c->out_dtype != FD_DTYPE_U8) return false;
  if (c->mlp_gated != 0 && c->mlp_gated != 1) return false;
  if (c->qk_norm != 0 && c->qk_norm != 1) return false;
  if (c->mlp_fp8 != 0 && c->mlp_fp8 != 1) return false;
  if (c->first_chunk_frames != 0 && c->first_chunk_frames != 1) return false;
  if (c->rope_mode != FD_ROPE_ABS && c->rope_mode != FD_ROPE_WINDOW_REL) return false;
  if (!(c->norm_eps >= 0.f) || !(c->rope_base > 1.f)) return false;
  const long long L = static_cast<long long>(c->latent_h / c->patch) * (c->latent_w / c->patch);
  if (L * c->r_t * c->window > (1LL << 26)) return false;
  return true;
}

Dims dims_of(const fd_config* c) {
  Dims d;
  d.C = c->latent_channels; d.H = c->latent_h; d.W = c->latent_w; d.p = c->patch;
  d.D = c->hidden; d.N = c->heads; d.G = c->kv_groups; d.Dh = kHeadDim; d.Mr = c->mlp_ratio;
  d.nb = c->n_blocks; d.nr = c->n_refine; d.Wn = c->window; d.rt = c->r_t;
  d.rs = c->vae_spatial * c->patch; d.Cout = c->out_channels;
  d.cin = d.C * d.p * d.p; d.gh = d.H / d.p; d.gw = d.W / d.p; d.L = d.gh * d.gw;
  d.head_out = d.Cout * d.rs * d.rs; d.qkv_out = (d.N + 2 * d.G) * kHeadDim;
  d.u8 = c->out_dtype == FD_DTYPE_U8;
  d.gated = c->mlp_gated == 1;
  d.qk = c->qk_norm == 1;
  d.fp8 = c->mlp_fp8 == 1;
  d.f1 = c->first_chunk_frames == 1;
  return d;
}

bool same_cfg(const fd_config* a, const fd_config* b) {
  return std::memcmp(a, b, sizeof(fd_config)) == 0;
}

// blob element counts, in blob order
struct BlobEntry {
  size_t elems;
  int kind;          // 0 weight (bf16 on device), 1 fp32, 2 weight (e4m3 on device, one
                     // power-of-two scale per row of row_len elements)
  size_t gate_rows;  // > 0: gated MLP layer 1 (gate rows, then as many up rows) whose rows the
  size_t row_len;    // device copy interleaves in blocks of 32 (see gated_row)
};
void blob_layout(const Dims& d, std::vector<BlobEntry>& out) {
  auto W = [&](size_t n) { out.push_back({n, 0, 0, 0}); };
  auto F = [&](size_t n) { out.push_back({n, 1, 0, 0}); };
  const size_t D = d.D, Dm = static_cast<size_t>(d.Mr) * d.D;
  W(D * d.cin); F(D);
  auto block = [&] {
    F(D); W(static_cast<size_t>(d.qkv_out) * D); F(d.qkv_out); F(kHeadDim); F(kHeadDim);
    W(D * d.N * kHeadDim); F(D); F(D);
    if (d.gated) {
      out.push_back({2 * Dm * D, d.fp8 ? 2 : 0, Dm, D});
      out.push_back({2 * Dm, 1, Dm, 1});
    } else if (d.fp8) {
      out.push_back({Dm * D, 2, 0, D});
      F(Dm);
    } else {
      W(Dm * D); F(Dm);
    }
    if (d.fp8) {
      out.push_back({D * Dm, 2, 0, Dm});
    } else {
      W(D * Dm);
    }
    F(D);
  };
  for (int b = 0; b < d.nb; ++b) block();
  F(D); W(static_cast<size_t>(d.rt) * D * D); F(static_cast<size_t>(d.rt) * D);
  for (int b = 0; b < d.nr; ++b) block();
  F(D); W(D * D); F(D); W(static_cast<size_t>(d.head_out) * D); F(d.head_out);
}

// Device row of blob row r of a gated MLP layer 1 with `gate` gate rows: the EPI_SWIGLU
// epilogue wants gate and up rows of the same 32 hidden units side by side (64-row blocks).
size_t gated_row(size_t r, size_t gate) {
  const size_t u = r < gate ? r : r - gate;
  return (u / 32) * 64 + (r < gate ? 0 : 32) + u % 32;
}

// smallest power of two >= x (x > 0), exactly
double pow2_ceil(double x) {
  int e = 0;
  const double m = std::frexp(x, &e);  // x = m 2^e, 0.5 <= m < 1
  return m == 0.5 ? std::ldexp(1.0, e - 1) : std::ldexp(1.0, e);
}

// value of an FP8 E4M3 code (OCP: sign, 4 exponent bits with bias 7, 3 mantissa bits;
// exponent 0 = subnormal, steps of 2^-9); the NaN codes never occur here
double e4m3_value(uint8_t c) {
  const int e = (c >> 3) & 15, m = c & 7;
  const double v = e == 0 ? std::ldexp(static_cast<double>(m), -9)
                          : std::ldexp(1.0 + m / 8.0, e - 7);
  return (c & 0x80) ? -v : v;
}

uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return 0x7FC0;  // NaN
  const uint32_t lsb = (u >> 16) & 1u;
  return static_cast<uint16_t>((u + 0x7FFFu + lsb) >> 16);
}
float bf16_to_f32(uint16_t b) {
  const uint32_t u = static_cast<uint32_t>(b) << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

// GEMM tile width for an M x N problem: a tile costs about (128 + BN) (a fixed part plus its
// width) and a persistent grid runs ceil(tiles / SMs) rounds; pick the cheapest, the wider tile
// on ties (the narrower one for epilogue-bound layers). Matches the measured best width on the
// decoder's shapes.
int pick_bn_step(int M, int N, int step, bool narrow_on_ties = false) {
  const int sms = num_sms();
  int best = 128;
  long long best_cost = -1;
  for (int bn : {64, 96, 128, 192, 256}) {
    if (bn % step) continue;
    if (bn == 64 && N > 64) continue;  // 64-wide tiles only for products that narrow
    const long long tiles = static_cast<long long>((M + 127) / 128) * ((N + bn - 1) / bn);
    const long long rounds = (tiles + sms - 1) / sms;
    const long long cost = rounds * (128 + bn);
    if (best_cost < 0 || cost < best_cost || (cost == best_cost && !narrow_on_ties)) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

struct Linear {
  __nv_bfloat16* w = nullptr;  // [N][K]
  float* b = nullptr;          // [N]
  int N = 0, K = 0, bn = 128;
  bool pair = false;           // 256-row tiles on CTA pairs (W boxes of bn / 2 rows)
  CUtensorMap tm;
};

// Launch shape of an M x N x K product. CTA pairs (256 x 256 tiles, each SM holding half of W)
// measured 4-10 % faster than the best single-CTA tile once there are at least 2.5 rounds of
// pair tiles, and slower on the smaller products, where a tile's fixed costs dominate; there
// the single-CTA width model of pick_bn_step (which matches the measured best width) decides.
struct TileChoice {
  int bn;
  bool pair;
};
TileChoice pick_tile(int M, int N, int K, int step, bool fp8, int force_pair = 0) {
  (void)K;
  (void)fp8;
  const int sms = num_sms();
  const long long pair_tiles = static_cast<long long>((M + 255) / 256) * ((N + 255) / 256);
  const bool pair = force_pair == 2 ||
                    (force_pair == 0 && 256 % step == 0 && 2 * pair_tiles >= 5LL * (sms / 2));
  if (pair) return {256, true};
  return {pick_bn_step(M, N, step), false};
}

struct LayerW {
  float *g1 = nullptr, *g2 = nullptr, *kg = nullptr, *vg = nullptr;
  Linear qkv, out, mlp1, mlp2;
  // FP8 MLP (mlp1 / mlp2 weights are e4m3): per-column dequantisation scales of the two
  // products and the reciprocal activation scales 1 / s_u, 1 / s_h
  float *cs1 = nullptr, *cs2 = nullptr;
  float inv_su = 1.f, inv_sh = 1.f;
};

}  // namespace

struct fd_weights_s {
  fd_config cfg;
  Dims d;
  void* arena = nullptr;
  std::vector<void*> entry;  // device address of every blob tensor, in blob order
  Linear embed, tup, head1, head2;
  float *g_f = nullptr, *g_h = nullptr;
  std::vector<LayerW> blocks, refine;
  int live_handles = 0;
};

namespace {

struct Ring {
  __nv_bfloat16* k = nullptr;   // [G][pitch][64]
  __half* vt = nullptr;         // [G][64][pitch] fp16
  CUtensorMap tm_k, tm_vt;      // attention loads
  CUtensorMap st_k, st_vt;      // QKV epilogue stores into ring slots
};

}  // namespace

struct fd_handle_s {
  fd_config cfg;
  Dims d;
  fd_weights w = nullptr;
  void* arena = nullptr;
  size_t arena_bytes = 0;
  int* state = nullptr;  // [0] chunk index t, [1] error bits
  int64_t t_host = 0;
  // unique for the life of the process: a destroyed handle's address can be reused by a new
  // one, so tables built for a set of handles remember serials, not addresses
  uint64_t serial = 0;
  bool error = false;
  cudaStream_t last_stream = nullptr;
  // fd_reset's clears, recorded on its stream; the next call that touches the handle's device
  // state on another stream waits for them (after_reset)
  cudaEvent_t ev_reset = nullptr;
  bool reset_pending = false;
  // fd_decode_chunks: a library-owned stream on which this handle's chunk runs beside the
  // other handles', forked from and joined back to the caller's stream (created on first use)
  cudaStream_t side = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  // activations (rows: L for the backbone, r_t L for refinement / head)
  __nv_bfloat16 *x0 = nullptr, *u = nullptr, *q = nullptr, *o = nullptr, *hid = nullptr;
  float *h = nullptr, *hf = nullptr, *F = nullptr;
  int pitchB = 0, pitchR = 0;
  std::vector<Ring> ringB, ringR;
  // attention key-range splits (fixed per stack for the steady-state window) and their
  // partial-result workspace
  int partsB = 1, partsR = 1;  // CTAs of the backbone / refinement attention launches
  float* attn_ws = nullptr;
  // temporal RoPE (cos, sin) of the current chunk: backbone frame, then the r_t refined frames
  float2* rope_tab = nullptr;
  // A-operand / Q descriptors
  CUtensorMap tm_x0, tm_uB, tm_uR, tm_oB, tm_oR, tm_hidB, tm_hidR, tm_hidH, tm_qB, tm_qR;
  CUtensorMap tm_q8B, tm_q8R;  // attention Q in 8-row boxes (tiles across two heads)
  // epilogue store descriptors
  CUtensorMap so_h, so_hf, so_tup, so_hidB, so_hidR, so_hidH, so_F, so_qB, so_qR;
  // FP8 MLP: e4m3 views of u (MLP input) and hid (MLP hidden), A operands and store map
  CUtensorMap tm_u8B, tm_u8R, tm_hid8B, tm_hid8R, so_hid8B, so_hid8R;
  // host-buffer decode: library-owned device copies of the latent and the pixels
  float* latent_buf = nullptr;
  void* pixel_buf = nullptr;
  // fd_decode_sequence_host (created on first use): a copy stream, the second latent / pixel
  // buffers, and per buffer the events latent in, chunk decoded, pixels out
  cudaStream_t copy = nullptr;
  float* latent_buf2 = nullptr;
  void* pixel_buf2 = nullptr;
  cudaEvent_t ev_cfork = nullptr, ev_in[2] = {}, ev_done[2] = {}, ev_out[2] = {};
  // tracing: launch count and, while profiling, one event pair per launch
  int64_t launches = 0;
  bool profiling = false;
  std::vector<cudaEvent_t> ev_start, ev_stop;
  std::vector<int> ev_kind;
  size_t ev_used = 0;
};

// Batched decode of independent streams (fd_decode_batch): the streams' tokens are stacked,
// each stream's rows padded to a multiple of 128 (Lp per frame), so that every GEMM runs once
// on all of them and no tile or 32-row slab holds two streams; attention and the pixel head
// run per stream on the streams' own caches.
struct fd_batch_s {
  fd_config cfg;
  Dims d;
  fd_weights w = nullptr;
  int nmax = 0, Lp = 0, Rp = 0;  // streams; padded rows per stream (backbone, refinement)
  void* arena = nullptr;
  __nv_bfloat16 *x0 = nullptr, *u = nullptr, *q = nullptr, *o = nullptr, *hid = nullptr;
  float *h = nullptr, *hf = nullptr, *F = nullptr, *attn_ws = nullptr;
  float2* rope = nullptr;               // [nmax][(1 + r_t) band_t] temporal RoPE per stream
  fd::QkvStream* table = nullptr;       // [n_blocks + n_refine][nmax] on the device
  fd::QkvStream* table_host = nullptr;  // pinned copy
  fd::AttnStream* attn_table = nullptr;       // [n_blocks + n_refine][nmax]: rings' K / V maps
  fd::AttnStream* attn_table_host = nullptr;  // pinned copy
  std::vector<uint64_t> table_for;      // serials of the handles the tables were written for
  size_t ws_stride = 0;                 // attention workspace floats per stream
  CUtensorMap tm_x0, tm_uB, tm_uR, tm_oB, tm_oR, tm_hidB, tm_hidR, tm_hidH;
  CUtensorMap so_h, so_hf, so_tup, so_hidB, so_hidR, so_hidH, so_F, so_qB, so_qR;
  CUtensorMap tm_u8B, tm_u8R, tm_hid8B, tm_hid8R, so_hid8B, so_hid8R;
  CUtensorMap tm_qB, tm_q8B, tm_qR, tm_q8R;  // stacked Q in boxes of 128 and 8 rows
  // the weights' products with launch shapes re-chosen for the stacked row counts (same
  // device weights; only the tile width, CTA pairing and W descriptor differ)
  Linear embed, tup, head1, head2;
  std::vector<LayerW> blocks, refine;
};

namespace {

double rope_inv_freq(int i, int band_t, int band_s, double base) {
  // pair i: temporal band (2*band_t dims) first, then row and column bands (2*band_s each)
  int j, d;
  if (i < band_t) { j = i; d = 2 * band_t; }
  else if (i < band_t + band_s) { j = i - band_t; d = 2 * band_s; }
  else { j = i - band_t - band_s; d = 2 * band_s; }
  return std::pow(base, -2.0 * j / d);
}

void fill_rope(fd::QkvEpi& q, float base) {
  q.band_s = kHeadDim / 6;                 // pairs per spatial band (10 at D_h = 64)
  q.band_t = kHeadDim / 2 - 2 * q.band_s;  // temporal pairs (12)
  for (int i = 0; i < fd::kRopePairs; ++i)
    q.inv_freq_s[i] =
        static_cast<float>(rope_inv_freq(i, q.band_t, q.band_s, static_cast<double>(base)));
}

int rope_band_t() { return kHeadDim / 2 - 2 * (kHeadDim / 6); }

void temporal_inv_freq(float base, double* out) {
  const int bt = rope_band_t(), bs = kHeadDim / 6;
  for (int i = 0; i < bt; ++i) out[i] = rope_inv_freq(i, bt, bs, static_cast<double>(base));
}

fd_status launch_ok(cudaError_t e) { return e == cudaSuccess ? FD_OK : FD_ERR_CUDA; }

// Launch one kernel of the decode path: counts it and, while profiling, brackets it with a
// pair of CUDA events on its stream.
template <class Fn>
fd_status traced(fd_handle h, int kind, cudaStream_t s, Fn&& fn) {
  size_t slot = 0;
  if (h->profiling) {
    slot = h->ev_used++;
    if (slot == h->ev_start.size()) {
      cudaEvent_t a, b;
      if (cudaEventCreate(&a) != cudaSuccess) return FD_ERR_CUDA;
      if (cudaEventCreate(&b) != cudaSuccess) {
        cudaEventDestroy(a);
        return FD_ERR_CUDA;
      }
      h->ev_start.push_back(a);
      h->ev_stop.push_back(b);
      h->ev_kind.push_back(kind);
    }
    h->ev_kind[slot] = kind;
    if (cudaEventRecord(h->ev_start[slot], s) != cudaSuccess) return FD_ERR_CUDA;
  }
  const fd_status st = launch_ok(fn());
  if (st != FD_OK) return st;
  h->launches++;
  if (h->profiling && cudaEventRecord(h->ev_stop[slot], s) != cudaSuccess) return FD_ERR_CUDA;
  return FD_OK;
}

// tile pairs the attention counters must cover (the larger of backbone and refinement)
static int attn_pairs(const Dims& d) {
  const int a = fd::attention_units(d.L, d.N, d.G);
  const int b = d.nr > 0 ? fd::attention_units(d.rt * d.L, d.N, d.G) : 0;
  return a > b ? a : b;
}

// CTAs of an attention of Lq rows over n_keys keys
int choose_parts(int Lq, int heads, int groups, int n_keys) {
  return fd::attention_parts(fd::attention_units(Lq, heads, groups), (n_keys + 127) / 128,
                             num_sms());
}

fd_status run_linear(fd_handle h, int kind, const CUtensorMap& tmA, const Linear& lin, int M,
                     fd::GemmParams p, const CUtensorMap& tmO, cudaStream_t s,
                     const CUtensorMap* tmK = nullptr, const CUtensorMap* tmV = nullptr) {
  p.M = M;
  p.N = lin.N;
  p.K = lin.K;
  p.bias = lin.b;
  p.err = h->state + 1;
  p.w_static = 1;  // written once by fd_weights_create (synchronous copy)
  const CUtensorMap& k = tmK ? *tmK : tmO;
  const CUtensorMap& v = tmV ? *tmV : tmO;
  return traced(h, kind, s, [&] {
    return fd::launch_gemm(tmA, lin.tm, tmO, k, v, p, lin.bn, lin.pair, num_sms(), s);
  });
}

fd_status run_norm(fd_handle h, const float* x, const float* g, int rows, cudaStream_t s) {
  const int D = h->d.D;
  const float eps = h->cfg.norm_eps;
  __nv_bfloat16* u = h->u;
  return traced(h, FD_K_RMSNORM, s, [&] { return fd::launch_rmsnorm(x, g, rows, D, eps, u, s); });
}

// one Transformer block (Sec. 3.2) on `rows` tokens of residual stream hbuf, with ring r
fd_status run_block(fd_handle h, const LayerW& lw, Ring& r, float* hbuf, int rows, int fpc,
                    int pitch, const CUtensorMap& tm_u, const CUtensorMap& tm_q,
                    const CUtensorMap& tm_o, const CUtensorMap& tm_hid, const CUtensorMap& so_h,
                    const CUtensorMap& so_q, const CUtensorMap& so_hid, bool refine,
                    cudaStream_t s) {
  const Dims& d = h->d;
  fd_status st;
  if ((st = run_norm(h, hbuf, lw.g1, rows, s))) return st;
  fd::GemmParams p{};
  p.epi = fd::EPI_QKV;
  fd::QkvEpi& q = p.qkv;
  q.heads = d.N; q.groups = d.G; q.knorm_g = lw.kg; q.vnorm_g = lw.vg; q.q_out = h->q;
  q.qk_norm = d.qk ? 1 : 0;
  q.k_ring = r.k; q.vt_ring = r.vt; q.ring_pitch = pitch; q.tokens = d.L; q.grid_w = d.gw;
  q.frames_per_chunk = fpc; q.window = d.Wn; q.step_dev = h->state; q.step_host = 0;
  q.eps = h->cfg.norm_eps;
  fill_rope(q, h->cfg.rope_base);
  q.rope_t = h->rope_tab + (refine ? q.band_t : 0);
  p.v_tma = rows % 8 == 0 ? 1 : 0;
  if ((st = run_linear(h, FD_K_QKV, tm_u, lw.qkv, rows, p, so_q, s, &r.st_k, &r.st_vt)))
    return st;

  fd::AttnParams a{};
  a.Lq = rows; a.heads = d.N; a.groups = d.G; a.ring_pitch = pitch; a.rows_per_chunk = rows;
  a.window = d.Wn; a.step_dev = h->state; a.n_keys_host = 0; a.out = h->o;
  a.ld_out = d.N * kHeadDim; a.scale_log2 = static_cast<float>(1.4426950408889634 / 8.0);
  a.err = h->state + 1;
  a.lq_pad = fd::attention_lq_pad(rows);
  a.parts = refine ? h->partsR : h->partsB;
  fd::attention_workspace_split(h->attn_ws, a.parts, attn_pairs(d), a);
  if ((st = traced(h, refine ? FD_K_ATTN_R : FD_K_ATTN_B, s,
                   [&] {
                     return fd::launch_attention(tm_q, refine ? h->tm_q8R : h->tm_q8B, r.tm_k,
                                                 r.tm_vt, a, s);
                   })))
    return st;

  fd::GemmParams po{};
  po.epi = fd::EPI_RESID;
  po.out_f32 = hbuf;
  po.ld_out = d.D;
  if ((st = run_linear(h, FD_K_OUT, tm_o, lw.out, rows, po, so_h, s))) return st;
  if (d.fp8) {
    // FP8 MLP (Sec. 4.6): u8 = e4m3(RMSNorm(h) g / s_u); hid8 = e4m3(GELU(u8 W1 s_u s_w1 + b1)
    // / s_h); h += hid8 W2 s_h s_w2 + b2
    const float* gain = lw.g2;
    const float eps = h->cfg.norm_eps, inv_su = lw.inv_su;
    uint8_t* u8 = reinterpret_cast<uint8_t*>(h->u);
    const int D = d.D;
    if ((st = traced(h, FD_K_RMSNORM, s, [&] {
           return fd::launch_rmsnorm_e4m3(hbuf, gain, rows, D, eps, u8, inv_su, s);
         })))
      return st;
    fd::GemmParams p1{};
    p1.epi = d.gated ? fd::EPI_SWIGLU_F8 : fd::EPI_GELU_F8;
    p1.fp8 = 1;
    p1.col_scale = lw.cs1;
    p1.out_scale = lw.inv_sh;
    p1.out_f8 = reinterpret_cast<uint8_t*>(h->hid);
    p1.ld_out = d.Mr * d.D;
    if ((st = run_linear(h, FD_K_MLP1, refine ? h->tm_u8R : h->tm_u8B, lw.mlp1, rows, p1,
                         refine ? h->so_hid8R : h->so_hid8B, s)))
      return st;
    fd::GemmParams p2 = po;
    p2.fp8 = 1;
    p2.col_scale = lw.cs2;
    return run_linear(h, FD_K_MLP2, refine ? h->tm_hid8R : h->tm_hid8B, lw.mlp2, rows, p2, so_h,
                      s);
  }
  if ((st = run_norm(h, hbuf, lw.g2, rows, s))) return st;
  fd::GemmParams p1{};
  p1.epi = d.gated ? fd::EPI_SWIGLU : fd::EPI_GELU;
  p1.out_bf16 = h->hid;
  p1.ld_out = d.Mr * d.D;
  if ((st = run_linear(h, FD_K_MLP1, tm_u, lw.mlp1, rows, p1, so_hid, s))) return st;
  return run_linear(h, FD_K_MLP2, tm_hid, lw.mlp2, rows, po, so_h, s);
}

// Order a call on stream s after a pending fd_reset, whose clears ran on the stream of the
// handle's previous call: a wait on the reset's event when s is another stream.
fd_status after_reset(fd_handle h, cudaStream_t s) {
  if (!h->reset_pending) return FD_OK;
  if (s != h->last_stream && cudaStreamWaitEvent(s, h->ev_reset, 0) != cudaSuccess)
    return FD_ERR_CUDA;
  h->reset_pending = false;
  return FD_OK;
}

fd_status decode_one(fd_handle h, const float* latent, void* pixels, cudaStream_t s) {
  const Dims& d = h->d;
  const fd_weights w = h->w;
  fd_status st;
  {
    const int frames[2] = {1, d.rt};
    double inv[fd::kRopePairs];
    temporal_inv_freq(h->cfg.rope_base, inv);
    const int* step = h->state;
    float2* tab = h->rope_tab;
    if ((st = traced(h, FD_K_ROPE, s, [&] {
           return fd::launch_rope_table(step, 0, 2, frames, rope_band_t(), inv, tab, s);
         })))
      return st;
  }
  __nv_bfloat16* x0 = h->x0;
  if ((st = traced(h, FD_K_UNSHUFFLE, s,
                   [&] { return fd::launch_unshuffle(latent, d.C, d.H, d.W, d.p, x0, s); })))
    return st;
  fd::GemmParams pe{};
  pe.epi = fd::EPI_F32;
  pe.out_f32 = h->h;
  pe.ld_out = d.D;
  if ((st = run_linear(h, FD_K_EMBED, h->tm_x0, w->embed, d.L, pe, h->so_h, s))) return st;
  for (int b = 0; b < d.nb; ++b)
    if ((st = run_block(h, w->blocks[b], h->ringB[b], h->h, d.L, 1, h->pitchB, h->tm_uB, h->tm_qB,
                        h->tm_oB, h->tm_hidB, h->so_h, h->so_qB, h->so_hidB, false, s)))
      return st;
  // temporal upsampling: RMSNorm, Linear D -> r_t D, channel block tau -> refined frame tau
  if ((st = run_norm(h, h->h, w->g_f, d.L, s))) return st;
  fd::GemmParams pt{};
  pt.epi = fd::EPI_TUP;
  pt.out_f32 = h->hf;
  pt.tup_tokens = d.L;
  pt.tup_hidden = d.D;
  if ((st = run_linear(h, FD_K_TUP, h->tm_uB, w->tup, d.L, pt, h->so_tup, s))) return st;
  const int R = d.rt * d.L;
  for (int b = 0; b < d.nr; ++b)
    if ((st = run_block(h, w->refine[b], h->ringR[b], h->hf, R, d.rt, h->pitchR, h->tm_uR,
                        h->tm_qR, h->tm_oR, h->tm_hidR, h->so_hf, h->so_qR, h->so_hidR, true, s)))
      return st;
  // spatial upsampling head: RMSNorm, Linear D->D + GELU, Linear D -> C r_s^2, PixelShuffle
  if ((st = run_norm(h, h->hf, w->g_h, R, s))) return st;
  fd::GemmParams ph{};
  ph.epi = fd::EPI_GELU;
  ph.out_bf16 = h->hid;
  ph.ld_out = d.D;
  if ((st = run_linear(h, FD_K_HEAD1, h->tm_uR, w->head1, R, ph, h->so_hidH, s))) return st;
  // the causal frame count (Fig. 2): chunk 0 emits refined frame 0 only (rows 0 .. L-1 of F)
  const int frames = d.f1 && h->t_host == 0 ? 1 : d.rt;
  fd::GemmParams pf{};
  if (fd::gemm_pixel_epilogue_ok(w->head2.bn, w->head2.pair, d.rs)) {
    // the pixel shuffle, clamp (and uint8 code) in the product's epilogue: F is never stored
    pf.epi = fd::EPI_PIXEL;
    pf.pix = {pixels, d.u8 ? 1 : 0, frames, d.L, d.gh, d.gw, d.rs};
    if ((st = run_linear(h, FD_K_HEAD2, h->tm_hidH, w->head2, R, pf, h->so_F, s))) return st;
    int* state = h->state;
    return traced(h, FD_K_ADVANCE, s, [&] { return fd::launch_advance(state, s); });
  }
  pf.epi = fd::EPI_F32;
  pf.out_f32 = h->F;
  pf.ld_out = d.head_out;
  if ((st = run_linear(h, FD_K_HEAD2, h->tm_hidH, w->head2, R, pf, h->so_F, s))) return st;
  const float* F = h->F;
  if ((st = traced(h, FD_K_PIXEL, s, [&] {
         return fd::launch_pixel_head(F, frames, d.gh, d.gw, d.Cout, d.rs, d.u8 ? 1 : 0, pixels,
                                      s);
       })))
    return st;
  int* state = h->state;
  return traced(h, FD_K_ADVANCE, s, [&] { return fd::launch_advance(state, s); });
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Re-choose the launch shape of a product of the weights for M rows (as fd_weights_create
// does for one stream's rows); step: the epilogue's column step, e4m3: FP8 weight
bool retile(Linear& lin, int M, int step, bool e4m3) {
  if (e4m3) {
    lin.bn = pick_bn_step(M, lin.N, step, step == 128);
    lin.pair = false;
    return tmap_e4m3(&lin.tm, lin.w, lin.K, lin.N, lin.K, lin.bn);
  }
  const TileChoice t = pick_tile(M, lin.N, lin.K, step, false);
  lin.bn = t.bn;
  lin.pair = t.pair;
  return tmap_bf16(&lin.tm, lin.w, lin.K, lin.N, static_cast<uint64_t>(lin.K) * 2, fd::kBK,
                   lin.pair ? lin.bn / 2 : lin.bn);
}

bool retile_block(LayerW& lw, const Dims& d, int M) {
  bool ok = retile(lw.qkv, M, 64, false) && retile(lw.out, M, 32, false);
  if (d.fp8)
    return ok && retile(lw.mlp1, M, d.gated ? 256 : 128, true) && retile(lw.mlp2, M, 32, true);
  return ok && retile(lw.mlp1, M, d.gated ? 128 : 64, false) && retile(lw.mlp2, M, 32, false);
}

// CTAs per stream of a batched attention launch over n streams: the GPU's SMs shared out
// (the launch is persistent, one CTA per SM), at most one per (tile pair, key block) unit of
// the full window
int batch_parts(int Lq, int n_keys, const Dims& d, int n) {
  const long long units =
      static_cast<long long>(fd::attention_units(Lq, d.N, d.G)) * ((n_keys + 127) / 128);
  const int share = std::max(1, num_sms() / n);
  return static_cast<int>(std::min<long long>(share, std::max(1LL, units)));
}

// ---------------------------------------------------------------- batched decode
// One Transformer block on the stacked rows of n streams (see fd_batch_s): the GEMMs and the
// norms run once on n * rows_s rows; the QKV epilogue appends each stream's K / V to its own
// ring (padding rows append nothing); attention runs once per stream on its own cache.
fd_status batch_block(fd_batch b, fd_handle* hs, int n, int layer, bool refine, cudaStream_t s) {
  const Dims& d = b->d;
  fd_handle h0 = hs[0];  // launches of the stacked kernels are traced on the first stream
  const LayerW& lw = refine ? b->refine[layer] : b->blocks[layer];
  const int rows_s = refine ? b->Rp : b->Lp;
  const int M = n * rows_s;
  float* hbuf = refine ? b->hf : b->h;
  const int D = d.D;
  const float eps = h0->cfg.norm_eps;
  const uint64_t NQ = static_cast<uint64_t>(d.N) * kHeadDim;
  fd_status st;
  {
    const float* g1 = lw.g1;
    __nv_bfloat16* u = b->u;
    if ((st = traced(h0, FD_K_RMSNORM, s,
                     [&] { return fd::launch_rmsnorm(hbuf, g1, M, D, eps, u, s); })))
      return st;
  }
  fd::GemmParams p{};
  p.epi = fd::EPI_QKV;
  fd::QkvEpi& q = p.qkv;
  q.heads = d.N; q.groups = d.G; q.knorm_g = lw.kg; q.vnorm_g = lw.vg; q.q_out = b->q;
  q.qk_norm = d.qk ? 1 : 0;
  q.ring_pitch = refine ? h0->pitchR : h0->pitchB; q.tokens = d.L; q.grid_w = d.gw;
  q.frames_per_chunk = refine ? d.rt : 1; q.window = d.Wn; q.eps = eps;
  fill_rope(q, h0->cfg.rope_base);
  q.streams = n;
  q.stream_rows = rows_s;
  q.frame_rows = b->Lp;
  q.stream = b->table + static_cast<size_t>(refine ? d.nb + layer : layer) * b->nmax;
  p.v_tma = 0;
  const CUtensorMap& so_q = refine ? b->so_qR : b->so_qB;
  if ((st = run_linear(h0, FD_K_QKV, refine ? b->tm_uR : b->tm_uB, lw.qkv, M, p, so_q, s, &so_q,
                       &so_q)))
    return st;
  {  // one launch for all streams: grid y = stream, parts_s CTAs each
    const int pairs = std::max(fd::attention_units(d.L, d.N, d.G),
                               fd::attention_units(b->Rp, d.N, d.G));
    Ring& r0 = refine ? h0->ringR[layer] : h0->ringB[layer];
    fd::AttnParams a{};
    a.Lq = refine ? b->Rp : d.L;
    a.heads = d.N; a.groups = d.G; a.ring_pitch = q.ring_pitch;
    a.rows_per_chunk = refine ? d.rt * d.L : d.L;
    a.window = d.Wn; a.step_dev = h0->state; a.n_keys_host = 0;
    a.out = b->o;
    a.ld_out = static_cast<int>(NQ); a.scale_log2 = static_cast<float>(1.4426950408889634 / 8.0);
    a.err = h0->state + 1;
    a.lq_pad = fd::attention_lq_pad(a.Lq);
    a.parts = batch_parts(a.Lq, d.Wn * a.rows_per_chunk, d, n);
    fd::attention_workspace_split(b->attn_ws, a.parts, pairs, a);
    a.streams = b->attn_table + static_cast<size_t>(refine ? d.nb + layer : layer) * b->nmax;
    a.n_streams = n;
    a.q_rows_stream = rows_s;
    a.ws_stride = b->ws_stride;
    const CUtensorMap& tq = refine ? b->tm_qR : b->tm_qB;
    const CUtensorMap& tq8 = refine ? b->tm_q8R : b->tm_q8B;
    if ((st = traced(h0, refine ? FD_K_ATTN_R : FD_K_ATTN_B, s,
                     [&] { return fd::launch_attention(tq, tq8, r0.tm_k, r0.tm_vt, a, s); })))
      return st;
  }
  fd::GemmParams po{};
  po.epi = fd::EPI_RESID;
  po.out_f32 = hbuf;
  po.ld_out = D;
  const CUtensorMap& so_h = refine ? b->so_hf : b->so_h;
  if ((st = run_linear(h0, FD_K_OUT, refine ? b->tm_oR : b->tm_oB, lw.out, M, po, so_h, s)))
    return st;
  if (d.fp8) {  // as in run_block (Sec. 4.6)
    const float* gain = lw.g2;
    const float inv_su = lw.inv_su;
    uint8_t* u8 = reinterpret_cast<uint8_t*>(b->u);
    if ((st = traced(h0, FD_K_RMSNORM, s, [&] {
           return fd::launch_rmsnorm_e4m3(hbuf, gain, M, D, eps, u8, inv_su, s);
         })))
      return st;
    fd::GemmParams p1{};
    p1.epi = d.gated ? fd::EPI_SWIGLU_F8 : fd::EPI_GELU_F8;
    p1.fp8 = 1;
    p1.col_scale = lw.cs1;
    p1.out_scale = lw.inv_sh;
    p1.out_f8 = reinterpret_cast<uint8_t*>(b->hid);
    p1.ld_out = d.Mr * d.D;
    if ((st = run_linear(h0, FD_K_MLP1, refine ? b->tm_u8R : b->tm_u8B, lw.mlp1, M, p1,
                         refine ? b->so_hid8R : b->so_hid8B, s)))
      return st;
    fd::GemmParams p2 = po;
    p2.fp8 = 1;
    p2.col_scale = lw.cs2;
    return run_linear(h0, FD_K_MLP2, refine ? b->tm_hid8R : b->tm_hid8B, lw.mlp2, M, p2, so_h, s);
  }
  {
    const float* g2 = lw.g2;
    __nv_bfloat16* u = b->u;
    if ((st = traced(h0, FD_K_RMSNORM, s,
                     [&] { return fd::launch_rmsnorm(hbuf, g2, M, D, eps, u, s); })))
      return st;
  }
  fd::GemmParams p1{};
  p1.epi = d.gated ? fd::EPI_SWIGLU : fd::EPI_GELU;
  p1.out_bf16 = b->hid;
  p1.ld_out = d.Mr * d.D;
  if ((st = run_linear(h0, FD_K_MLP1, refine ? b->tm_uR : b->tm_uB, lw.mlp1, M, p1,
                       refine ? b->so_hidR : b->so_hidB, s)))
    return st;
  return run_linear(h0, FD_K_MLP2, refine ? b->tm_hidR : b->tm_hidB, lw.mlp2, M, po, so_h, s);
}

// Algorithm 1 for chunk t_i of each of n streams at once (streams may be at different t)
fd_status decode_batch(fd_batch b, fd_handle* hs, int n, const float* const* latents,
                       void* const* pixels, cudaStream_t s) {
  const Dims& d = b->d;
  const fd_weights w = b->w;
  fd_handle h0 = hs[0];
  fd_status st;
  const int bt = rope_band_t();
  for (int i = 0; i < n; ++i) {
    const int frames[2] = {1, d.rt};
    double inv[fd::kRopePairs];
    temporal_inv_freq(h0->cfg.rope_base, inv);
    const int* step = hs[i]->state;
    float2* tab = b->rope + static_cast<size_t>(i) * (1 + d.rt) * bt;
    if ((st = traced(hs[i], FD_K_ROPE, s, [&] {
           return fd::launch_rope_table(step, 0, 2, frames, bt, inv, tab, s);
         })))
      return st;
    __nv_bfloat16* x0 = b->x0 + static_cast<size_t>(i) * b->Lp * d.cin;
    const float* z = latents[i];
    if ((st = traced(hs[i], FD_K_UNSHUFFLE, s,
                     [&] { return fd::launch_unshuffle(z, d.C, d.H, d.W, d.p, x0, s); })))
      return st;
  }
  const int MB = n * b->Lp, MR = n * b->Rp;
  fd::GemmParams pe{};
  pe.epi = fd::EPI_F32;
  pe.out_f32 = b->h;
  pe.ld_out = d.D;
  if ((st = run_linear(h0, FD_K_EMBED, b->tm_x0, b->embed, MB, pe, b->so_h, s))) return st;
  for (int l = 0; l < d.nb; ++l)
    if ((st = batch_block(b, hs, n, l, false, s))) return st;
  {
    const float* g = w->g_f;
    __nv_bfloat16* u = b->u;
    float* hb = b->h;
    const int D = d.D;
    const float eps = h0->cfg.norm_eps;
    if ((st = traced(h0, FD_K_RMSNORM, s,
                     [&] { return fd::launch_rmsnorm(hb, g, MB, D, eps, u, s); })))
      return st;
  }
  fd::GemmParams pt{};
  pt.epi = fd::EPI_TUP;
  pt.out_f32 = b->hf;
  pt.tup_tokens = b->Lp;  // stream i's token l: row i Lp + l; refined: i Rp + tau Lp + l
  pt.tup_hidden = d.D;
  if ((st = run_linear(h0, FD_K_TUP, b->tm_uB, b->tup, MB, pt, b->so_tup, s))) return st;
  for (int l = 0; l < d.nr; ++l)
    if ((st = batch_block(b, hs, n, l, true, s))) return st;
  {
    const float* g = w->g_h;
    __nv_bfloat16* u = b->u;
    float* hb = b->hf;
    const int D = d.D;
    const float eps = h0->cfg.norm_eps;
    if ((st = traced(h0, FD_K_RMSNORM, s,
                     [&] { return fd::launch_rmsnorm(hb, g, MR, D, eps, u, s); })))
      return st;
  }
  fd::GemmParams ph{};
  ph.epi = fd::EPI_GELU;
  ph.out_bf16 = b->hid;
  ph.ld_out = d.D;
  if ((st = run_linear(h0, FD_K_HEAD1, b->tm_uR, b->head1, MR, ph, b->so_hidH, s))) return st;
  fd::GemmParams pf{};
  pf.epi = fd::EPI_F32;
  pf.out_f32 = b->F;
  pf.ld_out = d.head_out;
  if ((st = run_linear(h0, FD_K_HEAD2, b->tm_hidH, b->head2, MR, pf, b->so_F, s))) return st;
  for (int i = 0; i < n; ++i) {
    const float* F = b->F + static_cast<size_t>(i) * b->Rp * d.head_out;
    const int frames = d.f1 && hs[i]->t_host == 0 ? 1 : d.rt;
    void* pix = pixels[i];
    const int Lp = b->Lp;
    if ((st = traced(hs[i], FD_K_PIXEL, s, [&] {
           return fd::launch_pixel_head(F, frames, d.gh, d.gw, d.Cout, d.rs, d.u8 ? 1 : 0, pix, s,
                                        Lp);
         })))
      return st;
    int* state = hs[i]->state;
    if ((st = traced(hs[i], FD_K_ADVANCE, s, [&] { return fd::launch_advance(state, s); })))
      return st;
  }
  return FD_OK;
}



constexpr int kMaxAttnParts = 4096;  // CTAs of one attention launch (fd_op_attention)

}  // namespace

extern "C" {

const char* fd_status_str(fd_status s) {
  switch (s) {
    case FD_OK: return "ok";
    case FD_ERR_INVALID_ARG: return "invalid argument";
    case FD_ERR_CONFIG: return "unsupported configuration";
    case FD_ERR_OOM: return "device out of memory";
    case FD_ERR_CUDA: return "CUDA error";
    case FD_ERR_STATE: return "handle in error state (fd_reset it)";
    case FD_ERR_DEVICE_TIMEOUT: return "device wait timed out";
    case FD_ERR_UNSUPPORTED: return "device is not sm_103";
  }
  return "unknown status";
}

size_t fd_weights_blob_elems(const fd_config* cfg) {
  if (!valid_cfg(cfg)) return 0;
  std::vector<BlobEntry> e;
  blob_layout(dims_of(cfg), e);
  size_t n = 0;
  for (auto& x : e) n += x.elems;
  return n;
}

size_t fd_weights_blob_bytes(const fd_config* cfg, int blob_dtype) {
  if (blob_dtype != FD_DTYPE_F32 && blob_dtype != FD_DTYPE_BF16) return 0;
  return fd_weights_blob_elems(cfg) * (blob_dtype == FD_DTYPE_F32 ? 4 : 2);
}

size_t fd_latent_bytes(const fd_config* cfg) {
  if (!valid_cfg(cfg)) return 0;
  return static_cast<size_t>(cfg->latent_channels) * cfg->latent_h * cfg->latent_w * 4;
}

size_t fd_pixels_bytes(const fd_config* cfg) {
  if (!valid_cfg(cfg)) return 0;
  const Dims d = dims_of(cfg);
  return static_cast<size_t>(d.Cout) * d.rt * d.gh * d.rs * d.gw * d.rs * (d.u8 ? 1 : 4);
}

static size_t attn_ws_floats(const Dims& d) {
  const int R = d.rt * d.L;
  const int sB = choose_parts(d.L, d.N, d.G, d.Wn * d.L);
  const int sR = d.nr > 0 ? choose_parts(R, d.N, d.G, d.Wn * R) : 1;
  return fd::attention_workspace_floats(sB > sR ? sB : sR, attn_pairs(d));
}

static size_t handle_layout(const Dims& d, size_t* off /* 16 offsets */, int* pitchB,
                            int* pitchR) {
  const size_t R = static_cast<size_t>(d.rt) * d.L;
  *pitchB = static_cast<int>(align_up(static_cast<size_t>(d.Wn) * d.L, 128));
  *pitchR = static_cast<int>(align_up(static_cast<size_t>(d.Wn) * R, 128));
  size_t sizes[15] = {
      16,                                              // state
      static_cast<size_t>(d.L) * d.cin * 2,            // x0
      R * d.D * 2,                                     // u
      R * d.N * kHeadDim * 2,                          // q
      R * d.N * kHeadDim * 2,                          // o
      R * static_cast<size_t>(d.Mr) * d.D * 2,         // hid
      static_cast<size_t>(d.L) * d.D * 4,              // h
      R * d.D * 4,                                     // hf
      R * d.head_out * 4,                              // F
      static_cast<size_t>(d.nb) * 2 * d.G * *pitchB * kHeadDim * 2,  // backbone rings
      static_cast<size_t>(d.nr) * 2 * d.G * *pitchR * kHeadDim * 2,  // refinement rings
      static_cast<size_t>(d.C) * d.H * d.W * 4,                      // latent (host decode)
      static_cast<size_t>(d.Cout) * d.rt * d.gh * d.rs * d.gw * d.rs * (d.u8 ? 1 : 4),  // pixels
      attn_ws_floats(d) * 4,                                         // attention partials
      static_cast<size_t>(1 + d.rt) * kHeadDim / 2 * sizeof(float2),  // temporal RoPE table
  };
  size_t cur = 0;
  for (int i = 0; i < 15; ++i) {
    off[i] = cur;
    cur = align_up(cur + sizes[i], 1024);
  }
  off[15] = cur;
  return cur;
}

size_t fd_handle_device_bytes(const fd_config* cfg) {
  if (!valid_cfg(cfg)) return 0;
  size_t off[16];
  int a, b;
  return handle_layout(dims_of(cfg), off, &a, &b);
}

fd_status fd_weights_create(const fd_config* cfg, const void* host_blob, size_t blob_bytes,
                            int blob_dtype, fd_weights* out) {
  if (out == nullptr) return FD_ERR_INVALID_ARG;
  *out = nullptr;
  if (!valid_cfg(cfg)) return FD_ERR_CONFIG;
  if (host_blob == nullptr) return FD_ERR_INVALID_ARG;
  if (blob_dtype != FD_DTYPE_F32 && blob_dtype != FD_DTYPE_BF16) return FD_ERR_INVALID_ARG;
  if (blob_bytes != fd_weights_blob_bytes(cfg, blob_dtype)) return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  if (!load_encode()) return FD_ERR_CUDA;

  const Dims d = dims_of(cfg);
  std::vector<BlobEntry> layout;
  blob_layout(d, layout);
  // device arena: bf16 (or e4m3) weights and fp32 vectors in blob order, each 256-byte
  // aligned, then the FP8 column scales of every block (FP8 MLPs only)
  std::vector<size_t> doff(layout.size());
  size_t cur = 0;
  for (size_t i = 0; i < layout.size(); ++i) {
    doff[i] = cur;
    const size_t esz_dev = layout[i].kind == 0 ? 2 : (layout[i].kind == 1 ? 4 : 1);
    cur = align_up(cur + layout[i].elems * esz_dev, 256);
  }
  const size_t Dm = static_cast<size_t>(d.Mr) * d.D;
  const size_t fp8_cs_bytes =  // per block: mlp1 (gate and up when gated), mlp2 column scales
      align_up(((d.gated ? 2 : 1) * Dm + d.D) * 4, 256);
  const size_t fp8_off = cur;
  if (d.fp8) cur += static_cast<size_t>(d.nb + d.nr) * fp8_cs_bytes;
  std::vector<uint8_t> stage;
  std::vector<std::vector<double>> row_scale(layout.size()), row_norm(layout.size());
  try {
    stage.assign(cur, 0);
  } catch (...) {
    return FD_ERR_OOM;
  }
  auto blob_value = [&](size_t i) -> float {
    float f;
    if (blob_dtype == FD_DTYPE_F32) {
      std::memcpy(&f, static_cast<const uint8_t*>(host_blob) + 4 * i, 4);
    } else {
      uint16_t b;
      std::memcpy(&b, static_cast<const uint8_t*>(host_blob) + 2 * i, 2);
      f = bf16_to_f32(b);
    }
    return f;
  };
  size_t src = 0;
  for (size_t i = 0; i < layout.size(); ++i) {
    const BlobEntry& e = layout[i];
    if (e.kind == 2) {
      // FP8 weight (Sec. 4.6): per row, s = 2^ceil(log2(max|w| / 448)) and code = e4m3(w / s)
      // (round to nearest even; |w / s| <= 448, so nothing saturates). Keeps s and the norm of
      // the dequantised row for the static activation scales.
      // (row_scale in device row order, row_norm in blob row order; the gated layer's rows are
      // interleaved on the device like the bf16 one's)
      const size_t rows = e.elems / e.row_len;
      row_scale[i].resize(rows);
      row_norm[i].resize(rows);
      for (size_t r = 0; r < rows; ++r, src += e.row_len) {
        const size_t dr = e.gate_rows ? gated_row(r, e.gate_rows) : r;
        double amax = 0.0;
        for (size_t k = 0; k < e.row_len; ++k)
          amax = std::fmax(amax, std::fabs(static_cast<double>(blob_value(src + k))));
        const double sc = amax > 0.0 ? pow2_ceil(amax / 448.0) : 1.0;
        double ss = 0.0;
        for (size_t k = 0; k < e.row_len; ++k) {
          const float x = static_cast<float>(static_cast<double>(blob_value(src + k)) / sc);
          const uint8_t code = __nv_cvt_float_to_fp8(x, __NV_SATFINITE, __NV_E4M3);
          stage[doff[i] + dr * e.row_len + k] = code;
          const double dq = e4m3_value(code) * sc;
          ss += dq * dq;
        }
        row_scale[i][dr] = sc;
        row_norm[i][r] = std::sqrt(ss);
      }
      continue;
    }
    for (size_t k0 = 0; k0 < e.elems; ++k0, ++src) {
      const size_t k =
          e.gate_rows ? gated_row(k0 / e.row_len, e.gate_rows) * e.row_len + k0 % e.row_len : k0;
      const float f = blob_value(src);
      if (layout[i].kind == 0) {
        const uint16_t b = f32_to_bf16_rne(f);
        std::memcpy(&stage[doff[i] + 2 * k], &b, 2);
      } else {
        std::memcpy(&stage[doff[i] + 4 * k], &f, 4);
      }
    }
  }
  fd_weights w = new (std::nothrow) fd_weights_s;
  if (w == nullptr) return FD_ERR_OOM;
  w->cfg = *cfg;
  w->d = d;
  if (cudaMalloc(&w->arena, cur) != cudaSuccess) {
    delete w;
    return FD_ERR_OOM;
  }
  uint8_t* base = static_cast<uint8_t*>(w->arena);
  for (size_t i = 0; i < layout.size(); ++i) w->entry.push_back(base + doff[i]);
  size_t idx = 0;
  auto next = [&]() { return base + doff[idx++]; };
  auto host_f32 = [&](size_t entry) { return reinterpret_cast<const float*>(&stage[doff[entry]]); };
  int fp8_block = 0;
  // fp32_epi: the layer's epilogue stores fp32 (patch-embed, out-projection, MLP down, temporal
  // upsampling, head layer 2), which allows the narrower 96-wide tiles
  auto linear = [&](Linear& lin, int N, int K, int M, bool fp32_epi) -> bool {
    lin.w = reinterpret_cast<__nv_bfloat16*>(next());
    lin.b = reinterpret_cast<float*>(next());
    lin.N = N;
    lin.K = K;
    const TileChoice t = pick_tile(M, N, K, fp32_epi ? 32 : 64, false);
    lin.bn = t.bn;
    lin.pair = t.pair;
    return tmap_bf16(&lin.tm, lin.w, K, N, static_cast<uint64_t>(K) * 2, fd::kBK,
                     lin.pair ? lin.bn / 2 : lin.bn);
  };
  // FP8 linear: e4m3 weight [N][K] in boxes of 128 bytes (= 128 K elements)
  auto linear_e4m3 = [&](Linear& lin, int N, int K, int M, int step) -> bool {
    lin.w = reinterpret_cast<__nv_bfloat16*>(next());
    lin.b = reinterpret_cast<float*>(next());
    lin.N = N;
    lin.K = K;
    // the e4m3 GELU epilogue outweighs the FP8 MMAs: narrower tiles overlap it better
    lin.bn = pick_bn_step(M, N, step, step == 128);
    lin.pair = false;
    return tmap_e4m3(&lin.tm, lin.w, K, N, K, lin.bn);
  };
  bool ok = linear(w->embed, d.D, d.cin, d.L, true);
  auto block = [&](LayerW& lw, int M) {
    lw.g1 = reinterpret_cast<float*>(next());
    ok = ok && linear(lw.qkv, d.qkv_out, d.D, M, false);
    lw.kg = reinterpret_cast<float*>(next());
    lw.vg = reinterpret_cast<float*>(next());
    ok = ok && linear(lw.out, d.D, d.N * kHeadDim, M, true);
    const size_t e_g2 = idx;
    lw.g2 = reinterpret_cast<float*>(next());
    if (d.fp8) {
      // Static scales (Sec. 4.6 "static-calibrated"), from bounds no input can exceed:
      //   u = RMSNorm(h) g has |u_i| <= sqrt(D) max|g|          -> s_u = 2^ceil(log2(./448))
      //   |GELU(z_j)| <= max(1, |z_j|) and |z_j| <= 1.125 sqrt(D) max|g| ||w1_j|| + |b1_j|
      //   (with the e4m3 rounding of u, at most 1 + 2^-3)         -> s_h likewise
      // Columns are dequantised by s_u s_w1[n] (layer 1) and s_h s_w2[n] (layer 2).
      // Gated: |SiLU(x)| <= max(|x|, 0.28), so |SiLU(gate_j) up_j| <= max(B_gate_j, 0.28) B_up_j.
      const size_t e_w1 = idx, e_b1 = idx + 1, e_w2 = idx + 2;
      const size_t N1 = (d.gated ? 2 : 1) * Dm;
      ok = ok && linear_e4m3(lw.mlp1, static_cast<int>(N1), d.D, M, d.gated ? 256 : 128);
      ok = ok && linear_e4m3(lw.mlp2, d.D, static_cast<int>(Dm), M, 32);
      const float* g2 = host_f32(e_g2);
      const float* b1 = host_f32(e_b1);  // device (interleaved) order when gated
      double gmax = 0.0;
      for (int i = 0; i < d.D; ++i) gmax = std::fmax(gmax, std::fabs(static_cast<double>(g2[i])));
      const double sq = std::sqrt(static_cast<double>(d.D));
      const double s_u = pow2_ceil(sq * gmax / 448.0);
      // bound on |z_j| of blob row j
      auto bz = [&](size_t j) {
        const size_t dj = d.gated ? gated_row(j, Dm) : j;
        return 1.125 * sq * gmax * row_norm[e_w1][j] + std::fabs(static_cast<double>(b1[dj]));
      };
      double bound = 0.0;
      for (size_t j = 0; j < Dm; ++j)
        bound = std::fmax(bound, d.gated ? std::fmax(bz(j), 0.28) * bz(Dm + j) : bz(j));
      const double s_h = pow2_ceil(std::fmax(bound, 1.0) / 448.0);
      const size_t off = fp8_off + static_cast<size_t>(fp8_block++) * fp8_cs_bytes;
      float* cs = reinterpret_cast<float*>(&stage[off]);
      for (size_t n = 0; n < N1; ++n) cs[n] = static_cast<float>(s_u * row_scale[e_w1][n]);
      for (int n = 0; n < d.D; ++n) cs[N1 + n] = static_cast<float>(s_h * row_scale[e_w2][n]);
      lw.cs1 = reinterpret_cast<float*>(base + off);
      lw.cs2 = lw.cs1 + N1;
      lw.inv_su = static_cast<float>(1.0 / s_u);
      lw.inv_sh = static_cast<float>(1.0 / s_h);
      return;
    }
    ok = ok && linear(lw.mlp1, (d.gated ? 2 : 1) * d.Mr * d.D, d.D, M, false);
    if (d.gated) {  // EPI_SWIGLU works on 128-column steps
      const TileChoice t = pick_tile(M, lw.mlp1.N, d.D, 128, false);
      lw.mlp1.bn = t.bn;
      lw.mlp1.pair = t.pair;
      ok = ok && tmap_bf16(&lw.mlp1.tm, lw.mlp1.w, d.D, lw.mlp1.N,
                           static_cast<uint64_t>(d.D) * 2, fd::kBK,
                           lw.mlp1.pair ? lw.mlp1.bn / 2 : lw.mlp1.bn);
    }
    ok = ok && linear(lw.mlp2, d.D, d.Mr * d.D, M, true);
  };
  w->blocks.resize(d.nb);
  for (auto& lw : w->blocks) block(lw, d.L);
  w->g_f = reinterpret_cast<float*>(next());
  ok = ok && linear(w->tup, d.rt * d.D, d.D, d.L, true);
  w->refine.resize(d.nr);
  for (auto& lw : w->refine) block(lw, d.rt * d.L);
  w->g_h = reinterpret_cast<float*>(next());
  ok = ok && linear(w->head1, d.D, d.D, d.rt * d.L, false);
  ok = ok && linear(w->head2, d.head_out, d.D, d.rt * d.L, true);
  if (!ok || idx != layout.size() ||
      cudaMemcpy(w->arena, stage.data(), cur, cudaMemcpyHostToDevice) != cudaSuccess) {
    cudaFree(w->arena);
    delete w;
    return FD_ERR_CUDA;
  }
  *out = w;
  return FD_OK;
}

fd_status fd_weights_destroy(fd_weights w) {
  if (w == nullptr) return FD_ERR_INVALID_ARG;
  if (w->live_handles > 0) return FD_ERR_STATE;
  cudaFree(w->arena);
  delete w;
  return FD_OK;
}

}  // extern "C"

// ---------------------------------------------------------------- hooks of the training step
namespace fd {

const fd_config* weights_config(fd_weights w) { return w ? &w->cfg : nullptr; }

size_t weights_entries(fd_weights w, const void** ptrs, size_t n) {
  if (w == nullptr) return 0;
  for (size_t i = 0; i < n && i < w->entry.size(); ++i) ptrs[i] = w->entry[i];
  return w->entry.size();
}

void weights_add_user(fd_weights w, int delta) {
  if (w) w->live_handles += delta;
}

cudaError_t scores_bwd(int M, int N, const __nv_bfloat16* Q, const __nv_bfloat16* dO, int ldq,
                       const __nv_bfloat16* K, const __nv_bfloat16* V, int ldk, const DsEpi& ds,
                       int* err, cudaStream_t s) {
  if (M < 1 || N < 32 || N % 32 || ldq % 8 || ldk % 8) return cudaErrorInvalidValue;
  CUtensorMap tq, tdo, tk, tv;
  if (!tmap_bf16(&tq, Q, kHeadDim, M, static_cast<uint64_t>(ldq) * 2, 64, 128) ||
      !tmap_bf16(&tdo, dO, kHeadDim, M, static_cast<uint64_t>(ldq) * 2, 64, 128) ||
      !tmap_bf16(&tk, K, kHeadDim, N, static_cast<uint64_t>(ldk) * 2, 64, 128) ||
      !tmap_bf16(&tv, V, kHeadDim, N, static_cast<uint64_t>(ldk) * 2, 64, 128))
    return cudaErrorInvalidValue;
  GemmParams p{};
  p.M = M; p.N = N; p.K = kHeadDim; p.epi = EPI_F32; p.err = err;
  p.ds = ds;
  return launch_gemm_scores_bwd(tq, tk, tdo, tv, p, num_sms(), s);
}

bool band_attention_maps(AttnStream* host, int T, int W, int rows_per_chunk, int G, int pitch,
                         const __nv_bfloat16* k, const __half* vt, const int* steps_dev,
                         int* err) {
  for (int i = 0; i < T; ++i) {
    const int j0 = i - W + 1 > 0 ? i - W + 1 : 0;
    const uint64_t key0 = static_cast<uint64_t>(j0) * rows_per_chunk;
    if ((key0 * 2) % 16 != 0 || key0 >= static_cast<uint64_t>(pitch)) return false;
    // K rows g pitch + key of the window, from its first key on
    if (!tmap_bf16(&host[i].k, k + key0 * kHeadDim, kHeadDim,
                   static_cast<uint64_t>(G) * pitch - key0, kHeadDim * 2, 64, 128))
      return false;
    // V^T [G 64][pitch] from column key0 on (the row pitch stays pitch)
    if (!tmap_f16(&host[i].vt, vt + key0, pitch - key0, static_cast<uint64_t>(G) * kHeadDim,
                  static_cast<uint64_t>(pitch) * 2, 64, 64))
      return false;
    host[i].step_dev = steps_dev + i;
    host[i].err = err;
  }
  return true;
}

bool attention_q_maps(CUtensorMap* q, CUtensorMap* q8, const __nv_bfloat16* base, int rows,
                      int heads) {
  const uint64_t NQ = static_cast<uint64_t>(heads) * kHeadDim;
  return tmap_bf16(q, base, NQ, rows, NQ * 2, 64, 128) &&
         tmap_bf16(q8, base, NQ, rows, NQ * 2, 64, 8);
}

cudaError_t gemm_view(int epi, int M, int N, int K, const __nv_bfloat16* A, int lda,
                      const __nv_bfloat16* W, int ldw, const float* bias, float* out, int ldo,
                      int* err, cudaStream_t s) {
  if ((epi != EPI_F32 && epi != EPI_RESID) || M < 1 || N < 1 || K < 1 || N % 32 || lda % 8 ||
      ldw % 8 || ldo % 4 || K > lda || K > ldw || N > ldo || !aligned16(A) || !aligned16(W) ||
      !aligned16(out) || !aligned16(bias))
    return cudaErrorInvalidValue;
  const TileChoice t = pick_tile(M, N, K, 32, false);
  CUtensorMap ta, tb, to;
  if (!tmap_bf16(&ta, A, K, M, static_cast<uint64_t>(lda) * 2, 64, 128) ||
      !tmap_bf16(&tb, W, K, N, static_cast<uint64_t>(ldw) * 2, 64, t.pair ? t.bn / 2 : t.bn) ||
      !tmap_out_f32(&to, out, N, M, ldo))
    return cudaErrorInvalidValue;
  GemmParams p{};
  p.M = M;
  p.N = N;
  p.K = K;
  p.epi = epi;
  p.bias = bias;
  p.out_f32 = out;
  p.ld_out = ldo;
  p.err = err;
  return launch_gemm(ta, tb, to, to, to, p, t.bn, t.pair, num_sms(), s);
}

}  // namespace fd

extern "C" {

fd_status fd_create(const fd_config* cfg, fd_weights w, fd_handle* out) {
  if (out == nullptr || w == nullptr) return FD_ERR_INVALID_ARG;
  *out = nullptr;
  if (!valid_cfg(cfg)) return FD_ERR_CONFIG;
  if (!same_cfg(cfg, &w->cfg)) return FD_ERR_CONFIG;
  fd_status st = check_device();
  if (st) return st;
  fd_handle h = new (std::nothrow) fd_handle_s;
  if (h == nullptr) return FD_ERR_OOM;
  static std::atomic<uint64_t> next_serial{0};
  h->serial = ++next_serial;
  h->cfg = *cfg;
  h->d = dims_of(cfg);
  h->w = w;
  const Dims& d = h->d;
  size_t off[16];
  h->arena_bytes = handle_layout(d, off, &h->pitchB, &h->pitchR);
  if (cudaMalloc(&h->arena, h->arena_bytes) != cudaSuccess) {
    delete h;
    return FD_ERR_OOM;
  }
  uint8_t* b = static_cast<uint8_t*>(h->arena);
  h->state = reinterpret_cast<int*>(b + off[0]);
  h->x0 = reinterpret_cast<__nv_bfloat16*>(b + off[1]);
  h->u = reinterpret_cast<__nv_bfloat16*>(b + off[2]);
  h->q = reinterpret_cast<__nv_bfloat16*>(b + off[3]);
  h->o = reinterpret_cast<__nv_bfloat16*>(b + off[4]);
  h->hid = reinterpret_cast<__nv_bfloat16*>(b + off[5]);
  h->h = reinterpret_cast<float*>(b + off[6]);
  h->hf = reinterpret_cast<float*>(b + off[7]);
  h->F = reinterpret_cast<float*>(b + off[8]);
  h->latent_buf = reinterpret_cast<float*>(b + off[11]);
  h->pixel_buf = b + off[12];
  h->attn_ws = reinterpret_cast<float*>(b + off[13]);
  h->rope_tab = reinterpret_cast<float2*>(b + off[14]);
  h->partsB = choose_parts(d.L, d.N, d.G, d.Wn * d.L);
  h->partsR = choose_parts(d.rt * d.L, d.N, d.G, d.Wn * d.rt * d.L);
  const size_t ringB_elems = static_cast<size_t>(d.G) * h->pitchB * kHeadDim;
  const size_t ringR_elems = static_cast<size_t>(d.G) * h->pitchR * kHeadDim;
  h->ringB.resize(d.nb);
  h->ringR.resize(d.nr);
  bool ok = true;
  for (int i = 0; i < d.nb; ++i) {
    Ring& r = h->ringB[i];
    r.k = reinterpret_cast<__nv_bfloat16*>(b + off[9]) + 2 * i * ringB_elems;
    r.vt = reinterpret_cast<__half*>(r.k + ringB_elems);
    ok = ok && tmap_bf16(&r.tm_k, r.k, kHeadDim, static_cast<uint64_t>(d.G) * h->pitchB,
                         kHeadDim * 2, 64, 128);
    ok = ok && tmap_f16(&r.tm_vt, r.vt, h->pitchB, static_cast<uint64_t>(d.G) * kHeadDim,
                         static_cast<uint64_t>(h->pitchB) * 2, 64, 64);
    ok = ok && tmap_kring_store(&r.st_k, r.k, d.L, d.Wn, d.G, h->pitchB);
    if (d.L % 8 == 0) ok = ok && tmap_vring_store(&r.st_vt, r.vt, d.L, d.Wn, d.G, h->pitchB);
    else r.st_vt = r.st_k;
  }
  for (int i = 0; i < d.nr; ++i) {
    Ring& r = h->ringR[i];
    r.k = reinterpret_cast<__nv_bfloat16*>(b + off[10]) + 2 * i * ringR_elems;
    r.vt = reinterpret_cast<__half*>(r.k + ringR_elems);
    ok = ok && tmap_bf16(&r.tm_k, r.k, kHeadDim, static_cast<uint64_t>(d.G) * h->pitchR,
                         kHeadDim * 2, 64, 128);
    ok = ok && tmap_f16(&r.tm_vt, r.vt, h->pitchR, static_cast<uint64_t>(d.G) * kHeadDim,
                         static_cast<uint64_t>(h->pitchR) * 2, 64, 64);
    const uint64_t R = static_cast<uint64_t>(d.rt) * d.L;
    ok = ok && tmap_kring_store(&r.st_k, r.k, R, d.Wn, d.G, h->pitchR);
    if (R % 8 == 0) ok = ok && tmap_vring_store(&r.st_vt, r.vt, R, d.Wn, d.G, h->pitchR);
    else r.st_vt = r.st_k;
  }
  const uint64_t R = static_cast<uint64_t>(d.rt) * d.L;
  const uint64_t NQ = static_cast<uint64_t>(d.N) * kHeadDim;
  const uint64_t Dm = static_cast<uint64_t>(d.Mr) * d.D;
  ok = ok && tmap_bf16(&h->tm_x0, h->x0, d.cin, d.L, d.cin * 2, 64, 128);
  ok = ok && tmap_bf16(&h->tm_uB, h->u, d.D, d.L, d.D * 2, 64, 128);
  ok = ok && tmap_bf16(&h->tm_uR, h->u, d.D, R, d.D * 2, 64, 128);
  ok = ok && tmap_bf16(&h->tm_oB, h->o, NQ, d.L, NQ * 2, 64, 128);
  ok = ok && tmap_bf16(&h->tm_oR, h->o, NQ, R, NQ * 2, 64, 128);
  ok = ok && tmap_bf16(&h->tm_qB, h->q, NQ, d.L, NQ * 2, 64, 128);
  ok = ok && tmap_bf16(&h->tm_qR, h->q, NQ, R, NQ * 2, 64, 128);
  ok = ok && tmap_bf16(&h->tm_q8B, h->q, NQ, d.L, NQ * 2, 64, 8);
  ok = ok && tmap_bf16(&h->tm_q8R, h->q, NQ, R, NQ * 2, 64, 8);
  ok = ok && tmap_bf16(&h->tm_hidB, h->hid, Dm, d.L, Dm * 2, 64, 128);
  ok = ok && tmap_bf16(&h->tm_hidR, h->hid, Dm, R, Dm * 2, 64, 128);
  ok = ok && tmap_bf16(&h->tm_hidH, h->hid, d.D, R, static_cast<uint64_t>(d.D) * 2, 64, 128);
  ok = ok && tmap_out_f32(&h->so_h, h->h, d.D, d.L, d.D);
  ok = ok && tmap_out_f32(&h->so_hf, h->hf, d.D, R, d.D);
  ok = ok && tmap_out_tup(&h->so_tup, h->hf, d.D, d.L, d.rt);
  ok = ok && tmap_out_bf16(&h->so_hidB, h->hid, Dm, d.L, Dm);
  ok = ok && tmap_out_bf16(&h->so_hidR, h->hid, Dm, R, Dm);
  ok = ok && tmap_out_bf16(&h->so_hidH, h->hid, d.D, R, d.D);
  ok = ok && tmap_out_f32(&h->so_F, h->F, d.head_out, R, d.head_out);
  ok = ok && tmap_out_bf16(&h->so_qB, h->q, NQ, d.L, NQ);
  ok = ok && tmap_out_bf16(&h->so_qR, h->q, NQ, R, NQ);
  if (d.fp8) {
    ok = ok && tmap_e4m3(&h->tm_u8B, h->u, d.D, d.L, d.D, 128);
    ok = ok && tmap_e4m3(&h->tm_u8R, h->u, d.D, R, d.D, 128);
    ok = ok && tmap_e4m3(&h->tm_hid8B, h->hid, Dm, d.L, Dm, 128);
    ok = ok && tmap_e4m3(&h->tm_hid8R, h->hid, Dm, R, Dm, 128);
    ok = ok && tmap_out_e4m3(&h->so_hid8B, h->hid, Dm, d.L, Dm);
    ok = ok && tmap_out_e4m3(&h->so_hid8R, h->hid, Dm, R, Dm);
  }
  if (!ok || cudaMemset(h->arena, 0, h->arena_bytes) != cudaSuccess ||
      cudaDeviceSynchronize() != cudaSuccess) {
    cudaFree(h->arena);
    delete h;
    return FD_ERR_CUDA;
  }
  w->live_handles++;
  *out = h;
  return FD_OK;
}

fd_status fd_decode_chunk(fd_handle h, const float* latent_dev, void* pixels_dev, void* stream) {
  if (h == nullptr || latent_dev == nullptr || pixels_dev == nullptr) return FD_ERR_INVALID_ARG;
  if (!aligned16(latent_dev) || !aligned16(pixels_dev)) return FD_ERR_INVALID_ARG;
  if (h->error) return FD_ERR_STATE;
  if (h->t_host >= (1LL << 30)) return FD_ERR_STATE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (after_reset(h, s) != FD_OK) return FD_ERR_CUDA;
  h->last_stream = s;
  fd_status st = decode_one(h, latent_dev, pixels_dev, s);
  if (st != FD_OK) {
    h->error = true;
    return st;
  }
  h->t_host++;
  return FD_OK;
}

fd_status fd_decode_chunks(fd_handle* hs, int n, const float* const* latents_dev,
                           void* const* pixels_dev, void* stream) {
  if (hs == nullptr || n < 0 || (n > 0 && (latents_dev == nullptr || pixels_dev == nullptr)))
    return FD_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i) {  // check everything before enqueueing anything
    fd_handle h = hs[i];
    if (h == nullptr || latents_dev[i] == nullptr || pixels_dev[i] == nullptr)
      return FD_ERR_INVALID_ARG;
    if (!aligned16(latents_dev[i]) || !aligned16(pixels_dev[i])) return FD_ERR_INVALID_ARG;
    for (int j = 0; j < i; ++j)
      if (hs[j] == h) return FD_ERR_INVALID_ARG;
    if (h->error || h->t_host >= (1LL << 30)) return FD_ERR_STATE;
    if (h->side == nullptr &&
        (cudaStreamCreateWithFlags(&h->side, cudaStreamNonBlocking) != cudaSuccess ||
         cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
         cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming) != cudaSuccess))
      return FD_ERR_CUDA;
  }
  if (n == 1) return fd_decode_chunk(hs[0], latents_dev[0], pixels_dev[0], stream);
  // fork: every handle's side stream starts after the work already on the caller's stream;
  // join: the caller's stream continues once every chunk is done. The independent streams'
  // kernels fill each other's launch gaps and idle SMs.
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (n > 0 && cudaEventRecord(hs[0]->ev_fork, s) != cudaSuccess) return FD_ERR_CUDA;
  for (int i = 0; i < n; ++i) {
    fd_handle h = hs[i];
    if (cudaStreamWaitEvent(h->side, hs[0]->ev_fork, 0) != cudaSuccess) return FD_ERR_CUDA;
    if (after_reset(h, h->side) != FD_OK) return FD_ERR_CUDA;
    fd_status st = decode_one(h, latents_dev[i], pixels_dev[i], h->side);
    if (st == FD_OK && cudaEventRecord(h->ev_join, h->side) != cudaSuccess) st = FD_ERR_CUDA;
    if (st != FD_OK) {
      h->error = true;
      return st;
    }
    h->t_host++;
    h->last_stream = s;  // ordered on the caller's stream once joined
  }
  for (int i = 0; i < n; ++i)
    if (cudaStreamWaitEvent(s, hs[i]->ev_join, 0) != cudaSuccess) return FD_ERR_CUDA;
  return FD_OK;
}

fd_status fd_batch_create(const fd_config* cfg, fd_weights w, int max_streams, fd_batch* out) {
  if (out == nullptr || w == nullptr || max_streams < 1 || max_streams > 64)
    return FD_ERR_INVALID_ARG;
  *out = nullptr;
  if (!valid_cfg(cfg) || !same_cfg(cfg, &w->cfg)) return FD_ERR_CONFIG;
  fd_status st = check_device();
  if (st) return st;
  fd_batch b = new (std::nothrow) fd_batch_s;
  if (b == nullptr) return FD_ERR_OOM;
  b->cfg = *cfg;
  b->d = dims_of(cfg);
  b->w = w;
  b->nmax = max_streams;
  const Dims& d = b->d;
  b->Lp = static_cast<int>(align_up(static_cast<size_t>(d.L), 128));
  b->Rp = d.rt * b->Lp;
  const size_t RB = static_cast<size_t>(max_streams) * b->Lp;  // stacked backbone rows
  const size_t RR = static_cast<size_t>(max_streams) * b->Rp;  // stacked refinement rows
  const uint64_t NQ = static_cast<uint64_t>(d.N) * kHeadDim;
  const uint64_t Dm = static_cast<uint64_t>(d.Mr) * d.D;
  const int bt = rope_band_t();
  const int pairs = std::max(fd::attention_units(d.L, d.N, d.G),
                             fd::attention_units(b->Rp, d.N, d.G));
  // per stream: partial results of up to one CTA per SM (a batch of one stream)
  b->ws_stride = align_up(fd::attention_workspace_floats(num_sms(), pairs), 64);
  const size_t ws = b->ws_stride * max_streams;
  const size_t sizes[12] = {
      RB * d.cin * 2,                                                  // x0
      RR * d.D * 2,                                                    // u
      RR * NQ * 2,                                                     // q
      RR * NQ * 2,                                                     // o
      RR * Dm * 2,                                                     // hid
      RB * d.D * 4,                                                    // h
      RR * d.D * 4,                                                    // hf
      RR * d.head_out * 4,                                             // F
      ws * 4,                                                          // attention partials
      static_cast<size_t>(max_streams) * (1 + d.rt) * bt * sizeof(float2),  // RoPE tables
      static_cast<size_t>(d.nb + d.nr) * max_streams * sizeof(fd::QkvStream),  // stream table
      static_cast<size_t>(d.nb + d.nr) * max_streams * sizeof(fd::AttnStream)};  // ring maps
  size_t off[12], cur = 0;
  for (int i = 0; i < 12; ++i) {
    off[i] = cur;
    cur = align_up(cur + sizes[i], 1024);
  }
  if (cudaMalloc(&b->arena, cur) != cudaSuccess) {
    delete b;
    return FD_ERR_OOM;
  }
  if (cudaMallocHost(&b->table_host, sizes[10]) != cudaSuccess) {
    cudaFree(b->arena);
    delete b;
    return FD_ERR_OOM;
  }
  if (cudaMallocHost(&b->attn_table_host, sizes[11]) != cudaSuccess) {
    cudaFreeHost(b->table_host);
    cudaFree(b->arena);
    delete b;
    return FD_ERR_OOM;
  }
  uint8_t* a = static_cast<uint8_t*>(b->arena);
  b->x0 = reinterpret_cast<__nv_bfloat16*>(a + off[0]);
  b->u = reinterpret_cast<__nv_bfloat16*>(a + off[1]);
  b->q = reinterpret_cast<__nv_bfloat16*>(a + off[2]);
  b->o = reinterpret_cast<__nv_bfloat16*>(a + off[3]);
  b->hid = reinterpret_cast<__nv_bfloat16*>(a + off[4]);
  b->h = reinterpret_cast<float*>(a + off[5]);
  b->hf = reinterpret_cast<float*>(a + off[6]);
  b->F = reinterpret_cast<float*>(a + off[7]);
  b->attn_ws = reinterpret_cast<float*>(a + off[8]);
  b->rope = reinterpret_cast<float2*>(a + off[9]);
  b->table = reinterpret_cast<fd::QkvStream*>(a + off[10]);
  b->attn_table = reinterpret_cast<fd::AttnStream*>(a + off[11]);
  bool ok = true;
  b->embed = w->embed;
  b->tup = w->tup;
  b->head1 = w->head1;
  b->head2 = w->head2;
  b->blocks = w->blocks;
  b->refine = w->refine;
  ok = ok && retile(b->embed, static_cast<int>(RB), 32, false);
  ok = ok && retile(b->tup, static_cast<int>(RB), 32, false);
  ok = ok && retile(b->head1, static_cast<int>(RR), 64, false);
  ok = ok && retile(b->head2, static_cast<int>(RR), 32, false);
  for (auto& lw : b->blocks) ok = ok && retile_block(lw, d, static_cast<int>(RB));
  for (auto& lw : b->refine) ok = ok && retile_block(lw, d, static_cast<int>(RR));
  ok = ok && tmap_bf16(&b->tm_x0, b->x0, d.cin, RB, d.cin * 2, 64, 128);
  ok = ok && tmap_bf16(&b->tm_uB, b->u, d.D, RB, d.D * 2, 64, 128);
  ok = ok && tmap_bf16(&b->tm_uR, b->u, d.D, RR, d.D * 2, 64, 128);
  ok = ok && tmap_bf16(&b->tm_oB, b->o, NQ, RB, NQ * 2, 64, 128);
  ok = ok && tmap_bf16(&b->tm_oR, b->o, NQ, RR, NQ * 2, 64, 128);
  ok = ok && tmap_bf16(&b->tm_hidB, b->hid, Dm, RB, Dm * 2, 64, 128);
  ok = ok && tmap_bf16(&b->tm_hidR, b->hid, Dm, RR, Dm * 2, 64, 128);
  ok = ok && tmap_bf16(&b->tm_hidH, b->hid, d.D, RR, static_cast<uint64_t>(d.D) * 2, 64, 128);
  ok = ok && tmap_out_f32(&b->so_h, b->h, d.D, RB, d.D);
  ok = ok && tmap_out_f32(&b->so_hf, b->hf, d.D, RR, d.D);
  ok = ok && tmap_out_tup(&b->so_tup, b->hf, d.D, b->Lp, d.rt, max_streams);
  ok = ok && tmap_out_bf16(&b->so_hidB, b->hid, Dm, RB, Dm);
  ok = ok && tmap_out_bf16(&b->so_hidR, b->hid, Dm, RR, Dm);
  ok = ok && tmap_out_bf16(&b->so_hidH, b->hid, d.D, RR, d.D);
  ok = ok && tmap_out_f32(&b->so_F, b->F, d.head_out, RR, d.head_out);
  ok = ok && tmap_out_bf16(&b->so_qB, b->q, NQ, RB, NQ);
  ok = ok && tmap_out_bf16(&b->so_qR, b->q, NQ, RR, NQ);
  if (d.fp8) {
    ok = ok && tmap_e4m3(&b->tm_u8B, b->u, d.D, RB, d.D, 128);
    ok = ok && tmap_e4m3(&b->tm_u8R, b->u, d.D, RR, d.D, 128);
    ok = ok && tmap_e4m3(&b->tm_hid8B, b->hid, Dm, RB, Dm, 128);
    ok = ok && tmap_e4m3(&b->tm_hid8R, b->hid, Dm, RR, Dm, 128);
    ok = ok && tmap_out_e4m3(&b->so_hid8B, b->hid, Dm, RB, Dm);
    ok = ok && tmap_out_e4m3(&b->so_hid8R, b->hid, Dm, RR, Dm);
  }
  ok = ok && tmap_bf16(&b->tm_qB, b->q, NQ, RB, NQ * 2, 64, 128);
  ok = ok && tmap_bf16(&b->tm_q8B, b->q, NQ, RB, NQ * 2, 64, 8);
  ok = ok && tmap_bf16(&b->tm_qR, b->q, NQ, RR, NQ * 2, 64, 128);
  ok = ok && tmap_bf16(&b->tm_q8R, b->q, NQ, RR, NQ * 2, 64, 8);
  // padding rows start (and, being outputs of row-wise kernels on zero inputs, stay) finite
  if (!ok || cudaMemset(b->arena, 0, cur) != cudaSuccess || cudaDeviceSynchronize() != cudaSuccess) {
    cudaFreeHost(b->attn_table_host);
    cudaFreeHost(b->table_host);
    cudaFree(b->arena);
    delete b;
    return FD_ERR_CUDA;
  }
  w->live_handles++;
  *out = b;
  return FD_OK;
}

fd_status fd_decode_batch(fd_batch b, fd_handle* hs, int n, const float* const* latents_dev,
                          void* const* pixels_dev, void* stream) {
  if (b == nullptr || hs == nullptr || n < 1 || n > b->nmax || latents_dev == nullptr ||
      pixels_dev == nullptr)
    return FD_ERR_INVALID_ARG;
  for (int i = 0; i < n; ++i) {  // check everything before enqueueing anything
    fd_handle h = hs[i];
    if (h == nullptr || latents_dev[i] == nullptr || pixels_dev[i] == nullptr)
      return FD_ERR_INVALID_ARG;
    if (!aligned16(latents_dev[i]) || !aligned16(pixels_dev[i])) return FD_ERR_INVALID_ARG;
    if (h->w != b->w) return FD_ERR_CONFIG;
    for (int j = 0; j < i; ++j)
      if (hs[j] == h) return FD_ERR_INVALID_ARG;
    if (h->error || h->t_host >= (1LL << 30)) return FD_ERR_STATE;
  }
  const Dims& d = b->d;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the per-layer stream table (rings, counters, RoPE tables) for this set of handles
  bool same_set = b->table_for.size() == static_cast<size_t>(n);
  for (int i = 0; i < n && same_set; ++i) same_set = b->table_for[i] == hs[i]->serial;
  if (!same_set) {
    if (cudaStreamSynchronize(s) != cudaSuccess) return FD_ERR_CUDA;  // table not in use
    const int bt = rope_band_t();
    for (int l = 0; l < d.nb + d.nr; ++l)
      for (int i = 0; i < n; ++i) {
        const bool refine = l >= d.nb;
        const Ring& r = refine ? hs[i]->ringR[l - d.nb] : hs[i]->ringB[l];
        fd::QkvStream& e = b->table_host[static_cast<size_t>(l) * b->nmax + i];
        e.k_ring = r.k;
        e.vt_ring = r.vt;
        e.step_dev = hs[i]->state;
        e.rope_t = b->rope + static_cast<size_t>(i) * (1 + d.rt) * bt + (refine ? bt : 0);
        fd::AttnStream& m = b->attn_table_host[static_cast<size_t>(l) * b->nmax + i];
        m.k = r.tm_k;
        m.vt = r.tm_vt;
        m.step_dev = hs[i]->state;
        m.err = hs[i]->state + 1;
      }
    const size_t entries = static_cast<size_t>(d.nb + d.nr) * b->nmax;
    if (cudaMemcpyAsync(b->table, b->table_host, entries * sizeof(fd::QkvStream),
                        cudaMemcpyHostToDevice, s) != cudaSuccess ||
        cudaMemcpyAsync(b->attn_table, b->attn_table_host, entries * sizeof(fd::AttnStream),
                        cudaMemcpyHostToDevice, s) != cudaSuccess)
      return FD_ERR_CUDA;
    b->table_for.resize(n);
    for (int i = 0; i < n; ++i) b->table_for[i] = hs[i]->serial;
  }
  for (int i = 0; i < n; ++i)
    if (after_reset(hs[i], s) != FD_OK) return FD_ERR_CUDA;
  const fd_status st = decode_batch(b, hs, n, latents_dev, pixels_dev, s);
  for (int i = 0; i < n; ++i) {
    if (st != FD_OK) {
      hs[i]->error = true;
    } else {
      hs[i]->t_host++;
      hs[i]->last_stream = s;
    }
  }
  return st;
}

fd_status fd_batch_destroy(fd_batch b) {
  if (b == nullptr) return FD_ERR_INVALID_ARG;
  cudaDeviceSynchronize();
  cudaFreeHost(b->attn_table_host);
  cudaFreeHost(b->table_host);
  cudaFree(b->arena);
  if (b->w) b->w->live_handles--;
  delete b;
  return FD_OK;
}

fd_status fd_decode_chunk_host(fd_handle h, const float* latent_host, void* pixels_host,
                               void* stream) {
  if (h == nullptr || latent_host == nullptr || pixels_host == nullptr) return FD_ERR_INVALID_ARG;
  if (h->error) return FD_ERR_STATE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t lb = fd_latent_bytes(&h->cfg);
  const size_t pb = fd_pixels_bytes(&h->cfg) / (h->d.f1 && h->t_host == 0 ? h->d.rt : 1);
  if (cudaMemcpyAsync(h->latent_buf, latent_host, lb, cudaMemcpyHostToDevice, s) != cudaSuccess) {
    h->error = true;
    return FD_ERR_CUDA;
  }
  fd_status st = fd_decode_chunk(h, h->latent_buf, h->pixel_buf, stream);
  if (st != FD_OK) return st;
  if (cudaMemcpyAsync(pixels_host, h->pixel_buf, pb, cudaMemcpyDeviceToHost, s) != cudaSuccess) {
    h->error = true;
    return FD_ERR_CUDA;
  }
  return FD_OK;
}

// The copy stream, events and second buffers of fd_decode_sequence_host
static fd_status sequence_setup(fd_handle h) {
  if (h->copy != nullptr) return FD_OK;
  if (cudaMalloc(&h->latent_buf2, fd_latent_bytes(&h->cfg)) != cudaSuccess ||
      cudaMalloc(&h->pixel_buf2, fd_pixels_bytes(&h->cfg)) != cudaSuccess)
    return FD_ERR_OOM;
  cudaEvent_t* evs[7] = {&h->ev_cfork, &h->ev_in[0], &h->ev_in[1], &h->ev_done[0],
                         &h->ev_done[1], &h->ev_out[0], &h->ev_out[1]};
  for (cudaEvent_t* e : evs)
    if (cudaEventCreateWithFlags(e, cudaEventDisableTiming) != cudaSuccess) return FD_ERR_CUDA;
  if (cudaStreamCreateWithFlags(&h->copy, cudaStreamNonBlocking) != cudaSuccess)
    return FD_ERR_CUDA;
  return FD_OK;
}

fd_status fd_decode_sequence_host(fd_handle h, int n, const float* const* latents_host,
                                  void* const* pixels_host, void* stream) {
  if (h == nullptr || n < 0 || (n > 0 && (latents_host == nullptr || pixels_host == nullptr)))
    return FD_ERR_INVALID_ARG;
  for (int t = 0; t < n; ++t)
    if (latents_host[t] == nullptr || pixels_host[t] == nullptr) return FD_ERR_INVALID_ARG;
  if (h->error) return FD_ERR_STATE;
  if (h->t_host + n >= (1LL << 30)) return FD_ERR_STATE;
  if (n == 0) return FD_OK;
  fd_status st = sequence_setup(h);
  if (st != FD_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaStream_t c = h->copy;
  if (after_reset(h, s) != FD_OK) return FD_ERR_CUDA;
  h->last_stream = s;
  float* lat[2] = {h->latent_buf, h->latent_buf2};
  void* pix[2] = {h->pixel_buf, h->pixel_buf2};
  const size_t lb = fd_latent_bytes(&h->cfg);
  auto fail = [&](fd_status e) {
    h->error = true;
    return e;
  };
  auto ok = [](cudaError_t e) { return e == cudaSuccess; };
  // the copies start after the work already on the caller's stream (earlier users of the
  // buffers); chunk 0's latent goes in first
  if (!ok(cudaEventRecord(h->ev_cfork, s)) || !ok(cudaStreamWaitEvent(c, h->ev_cfork, 0)) ||
      !ok(cudaMemcpyAsync(lat[0], latents_host[0], lb, cudaMemcpyHostToDevice, c)) ||
      !ok(cudaEventRecord(h->ev_in[0], c)))
    return fail(FD_ERR_CUDA);
  for (int t = 0; t < n; ++t) {
    const int b = t & 1, nb = (t + 1) & 1;
    // the next latent, into the buffer chunk t-1 read, while chunk t decodes; it goes ahead of
    // chunk t's pixels on the copy stream
    if (t + 1 < n) {
      if ((t >= 1 && !ok(cudaStreamWaitEvent(c, h->ev_done[nb], 0))) ||
          !ok(cudaMemcpyAsync(lat[nb], latents_host[t + 1], lb, cudaMemcpyHostToDevice, c)) ||
          !ok(cudaEventRecord(h->ev_in[nb], c)))
        return fail(FD_ERR_CUDA);
    }
    // chunk t: its latent is in, and chunk t-2's pixels have left the buffer it writes
    if (!ok(cudaStreamWaitEvent(s, h->ev_in[b], 0)) ||
        (t >= 2 && !ok(cudaStreamWaitEvent(s, h->ev_out[b], 0))))
      return fail(FD_ERR_CUDA);
    const size_t pb = fd_pixels_bytes(&h->cfg) / (h->d.f1 && h->t_host == 0 ? h->d.rt : 1);
    if ((st = decode_one(h, lat[b], pix[b], s)) != FD_OK) return fail(st);
    h->t_host++;
    // its pixels out on the copy stream once it is decoded
    if (!ok(cudaEventRecord(h->ev_done[b], s)) || !ok(cudaStreamWaitEvent(c, h->ev_done[b], 0)) ||
        !ok(cudaMemcpyAsync(pixels_host[t], pix[b], pb, cudaMemcpyDeviceToHost, c)) ||
        !ok(cudaEventRecord(h->ev_out[b], c)))
      return fail(FD_ERR_CUDA);
  }
  // the caller's stream continues once every chunk's pixels are out
  if (!ok(cudaStreamWaitEvent(s, h->ev_out[(n - 1) & 1], 0)) ||
      (n >= 2 && !ok(cudaStreamWaitEvent(s, h->ev_out[n & 1], 0))))
    return fail(FD_ERR_CUDA);
  return FD_OK;
}

fd_status fd_reset(fd_handle h) {
  if (h == nullptr) return FD_ERR_INVALID_ARG;
  if (h->ev_reset == nullptr &&
      cudaEventCreateWithFlags(&h->ev_reset, cudaEventDisableTiming) != cudaSuccess)
    return FD_ERR_CUDA;
  if (cudaMemsetAsync(h->state, 0, 2 * sizeof(int), h->last_stream) != cudaSuccess)
    return FD_ERR_CUDA;
  // a launch stopped by an error may leave attention counters non-zero
  if (attn_ws_floats(h->d) > 0 &&
      cudaMemsetAsync(h->attn_ws, 0, sizeof(int) * attn_pairs(h->d), h->last_stream) !=
          cudaSuccess)
    return FD_ERR_CUDA;
  if (cudaEventRecord(h->ev_reset, h->last_stream) != cudaSuccess) return FD_ERR_CUDA;
  h->reset_pending = true;
  h->t_host = 0;
  h->error = false;
  return FD_OK;
}

fd_status fd_destroy(fd_handle h) {
  if (h == nullptr) return FD_ERR_INVALID_ARG;
  cudaStreamSynchronize(h->last_stream);
  if (h->side != nullptr) {
    cudaStreamSynchronize(h->side);
    cudaStreamDestroy(h->side);
  }
  if (h->ev_fork != nullptr) cudaEventDestroy(h->ev_fork);
  if (h->ev_reset != nullptr) cudaEventDestroy(h->ev_reset);
  if (h->copy != nullptr) {
    cudaStreamSynchronize(h->copy);
    cudaStreamDestroy(h->copy);
  }
  for (cudaEvent_t e : {h->ev_cfork, h->ev_in[0], h->ev_in[1], h->ev_done[0], h->ev_done[1],
                        h->ev_out[0], h->ev_out[1]})
    if (e != nullptr) cudaEventDestroy(e);
  cudaFree(h->latent_buf2);
  cudaFree(h->pixel_buf2);
  if (h->ev_join != nullptr) cudaEventDestroy(h->ev_join);
  for (size_t i = 0; i < h->ev_start.size(); ++i) {
    cudaEventDestroy(h->ev_start[i]);
    cudaEventDestroy(h->ev_stop[i]);
  }
  cudaFree(h->arena);
  if (h->w) h->w->live_handles--;
  delete h;
  return FD_OK;
}

fd_status fd_profile_enable(fd_handle h, int enable) {
  if (h == nullptr) return FD_ERR_INVALID_ARG;
  h->profiling = enable != 0;
  return FD_OK;
}

fd_status fd_profile_collect(fd_handle h, int64_t* launches, double* ms) {
  if (h == nullptr || launches == nullptr || ms == nullptr) return FD_ERR_INVALID_ARG;
  for (size_t i = 0; i < h->ev_used; ++i) {
    if (cudaEventSynchronize(h->ev_stop[i]) != cudaSuccess) return FD_ERR_CUDA;
    float t = 0.f;
    if (cudaEventElapsedTime(&t, h->ev_start[i], h->ev_stop[i]) != cudaSuccess) return FD_ERR_CUDA;
    const int k = h->ev_kind[i];
    if (k >= 0 && k < FD_K_COUNT) {
      launches[k] += 1;
      ms[k] += t;
    }
  }
  h->ev_used = 0;
  return FD_OK;
}

int64_t fd_launch_count(fd_handle h) { return h ? h->launches : -1; }

int64_t fd_chunk_index(fd_handle h) { return h ? h->t_host : -1; }

}  // extern "C"

namespace {
// Header of a saved streaming state; the rings follow (per backbone layer, then per refinement
// layer: K [G][pitch][64] bf16, then V^T [G][64][pitch] fp16).
struct StateHeader {
  char magic[8];
  int64_t version;
  int64_t t;
  int64_t payload_bytes;
  fd_config cfg;
};
constexpr char kStateMagic[8] = {'F', 'D', 'S', 'T', 'A', 'T', 'E', '\0'};
constexpr int64_t kStateVersion = 1;

size_t ring_bytes(const Dims& d, int pitch) {  // K or V^T of one layer
  return static_cast<size_t>(d.G) * pitch * kHeadDim * 2;
}
size_t state_payload(const Dims& d) {
  const int pitchB = static_cast<int>(align_up(static_cast<size_t>(d.Wn) * d.L, 128));
  const int pitchR = static_cast<int>(align_up(static_cast<size_t>(d.Wn) * d.rt * d.L, 128));
  return 2 * (d.nb * ring_bytes(d, pitchB) + d.nr * ring_bytes(d, pitchR));
}
}  // namespace

extern "C" {

size_t fd_state_bytes(const fd_config* cfg) {
  if (!valid_cfg(cfg)) return 0;
  return sizeof(StateHeader) + state_payload(dims_of(cfg));
}

fd_status fd_save_state(fd_handle h, void* host_buf, size_t bytes, void* stream) {
  if (h == nullptr || host_buf == nullptr) return FD_ERR_INVALID_ARG;
  if (bytes != fd_state_bytes(&h->cfg)) return FD_ERR_INVALID_ARG;
  if (h->error) return FD_ERR_STATE;
  StateHeader hd;
  std::memset(&hd, 0, sizeof(hd));
  std::memcpy(hd.magic, kStateMagic, 8);
  hd.version = kStateVersion;
  hd.t = h->t_host;
  hd.payload_bytes = static_cast<int64_t>(state_payload(h->d));
  hd.cfg = h->cfg;
  std::memcpy(host_buf, &hd, sizeof(hd));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* dst = static_cast<uint8_t*>(host_buf) + sizeof(hd);
  auto copy_out = [&](const std::vector<Ring>& rings, int pitch) -> bool {
    const size_t n = ring_bytes(h->d, pitch);
    for (const Ring& r : rings) {
      if (cudaMemcpyAsync(dst, r.k, n, cudaMemcpyDeviceToHost, s) != cudaSuccess) return false;
      dst += n;
      if (cudaMemcpyAsync(dst, r.vt, n, cudaMemcpyDeviceToHost, s) != cudaSuccess) return false;
      dst += n;
    }
    return true;
  };
  if (!copy_out(h->ringB, h->pitchB) || !copy_out(h->ringR, h->pitchR)) return FD_ERR_CUDA;
  return FD_OK;
}

fd_status fd_load_state(fd_handle h, const void* host_buf, size_t bytes, void* stream) {
  if (h == nullptr || host_buf == nullptr) return FD_ERR_INVALID_ARG;
  if (bytes != fd_state_bytes(&h->cfg)) return FD_ERR_INVALID_ARG;
  StateHeader hd;
  std::memcpy(&hd, host_buf, sizeof(hd));
  if (std::memcmp(hd.magic, kStateMagic, 8) != 0 || hd.version != kStateVersion ||
      hd.payload_bytes != static_cast<int64_t>(state_payload(h->d)) ||
      !same_cfg(&hd.cfg, &h->cfg) || hd.t < 0 || hd.t >= (1LL << 30))
    return FD_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (after_reset(h, s) != FD_OK) return FD_ERR_CUDA;
  const uint8_t* src = static_cast<const uint8_t*>(host_buf) + sizeof(hd);
  auto copy_in = [&](std::vector<Ring>& rings, int pitch) -> bool {
    const size_t n = ring_bytes(h->d, pitch);
    for (Ring& r : rings) {
      if (cudaMemcpyAsync(r.k, src, n, cudaMemcpyHostToDevice, s) != cudaSuccess) return false;
      src += n;
      if (cudaMemcpyAsync(r.vt, src, n, cudaMemcpyHostToDevice, s) != cudaSuccess) return false;
      src += n;
    }
    return true;
  };
  // device chunk index and a clear error word; pageable source: staged before the call returns
  const int st[2] = {static_cast<int>(hd.t), 0};
  if (!copy_in(h->ringB, h->pitchB) || !copy_in(h->ringR, h->pitchR) ||
      cudaMemcpyAsync(h->state, st, sizeof(st), cudaMemcpyHostToDevice, s) != cudaSuccess)
    return FD_ERR_CUDA;
  // as in fd_reset: an attention launch stopped by an error may have left pair counters set
  if (attn_ws_floats(h->d) > 0 &&
      cudaMemsetAsync(h->attn_ws, 0, sizeof(int) * attn_pairs(h->d), s) != cudaSuccess)
    return FD_ERR_CUDA;
  h->t_host = hd.t;
  h->error = false;
  h->last_stream = s;
  return FD_OK;
}

fd_status fd_sync_status(fd_handle h) {
  if (h == nullptr) return FD_ERR_INVALID_ARG;
  if (cudaStreamSynchronize(h->last_stream) != cudaSuccess) {
    h->error = true;
    return FD_ERR_CUDA;
  }
  int st[2] = {0, 0};
  if (cudaMemcpy(st, h->state, sizeof(st), cudaMemcpyDeviceToHost) != cudaSuccess) {
    h->error = true;
    return FD_ERR_CUDA;
  }
  if (st[1] != 0) {
    h->error = true;
    return FD_ERR_DEVICE_TIMEOUT;
  }
  return h->error ? FD_ERR_STATE : FD_OK;
}

fd_status fd_debug_wait_timeout(fd_handle h, unsigned int limit_us, void* stream) {
  if (h == nullptr || limit_us < 1 || limit_us > 100000) return FD_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (after_reset(h, s) != FD_OK) return FD_ERR_CUDA;
  if (fd::launch_wait_check(h->state + 1, 1000ull * limit_us, s) != cudaSuccess)
    return FD_ERR_CUDA;
  h->last_stream = s;
  return FD_OK;
}

fd_status fd_debug_read_ring(fd_handle h, int which, int layer, void* dst_host,
                             size_t dst_bytes) {
  if (h == nullptr || dst_host == nullptr) return FD_ERR_INVALID_ARG;
  const Dims& d = h->d;
  const std::vector<Ring>& rings = which == 0 ? h->ringB : h->ringR;
  if ((which != 0 && which != 1) || layer < 0 || layer >= static_cast<int>(rings.size()))
    return FD_ERR_INVALID_ARG;
  const int rows = which == 0 ? d.L : d.rt * d.L;
  const int pitch = which == 0 ? h->pitchB : h->pitchR;
  const size_t n = static_cast<size_t>(d.G) * d.Wn * rows * kHeadDim;
  if (dst_bytes < 2 * n * 2) return FD_ERR_INVALID_ARG;
  if (cudaStreamSynchronize(h->last_stream) != cudaSuccess) return FD_ERR_CUDA;
  std::vector<uint16_t> kbuf(static_cast<size_t>(d.G) * pitch * kHeadDim);
  std::vector<uint16_t> vbuf(kbuf.size());
  if (cudaMemcpy(kbuf.data(), rings[layer].k, kbuf.size() * 2, cudaMemcpyDeviceToHost) ||
      cudaMemcpy(vbuf.data(), rings[layer].vt, vbuf.size() * 2, cudaMemcpyDeviceToHost))
    return FD_ERR_CUDA;
  uint16_t* out = static_cast<uint16_t*>(dst_host);
  const size_t span = static_cast<size_t>(d.Wn) * rows;
  for (int g = 0; g < d.G; ++g)
    for (size_t r = 0; r < span; ++r)
      for (int c = 0; c < kHeadDim; ++c) {
        out[(g * span + r) * kHeadDim + c] = kbuf[(static_cast<size_t>(g) * pitch + r) * kHeadDim + c];
        out[n + (g * span + r) * kHeadDim + c] =
            vbuf[(static_cast<size_t>(g) * kHeadDim + c) * pitch + r];
      }
  return FD_OK;
}

// ---------------------------------------------------------------- kernel-level entry points

fd_status fd_op_linear(int epilogue, int M, int N, int K, const void* A, const void* W,
                       const float* bias, void* out, int tup_hidden, int bn, int* err_dev,
                       void* stream) {
  return fd_op_linear_tiled(epilogue, M, N, K, A, W, bias, out, tup_hidden, bn, bn ? 1 : 0,
                            err_dev, stream);
}

fd_status fd_op_linear_tiled(int epilogue, int M, int N, int K, const void* A, const void* W,
                             const float* bias, void* out, int tup_hidden, int bn, int pair,
                             int* err_dev, void* stream) {
  if (pair < 0 || pair > 2) return FD_ERR_INVALID_ARG;
  if (M < 1 || N < 1 || K < 1 || A == nullptr || W == nullptr || bias == nullptr ||
      out == nullptr || err_dev == nullptr)
    return FD_ERR_INVALID_ARG;
  if (N % 32 || K % 8 || !aligned16(A) || !aligned16(W) || !aligned16(out) || !aligned16(bias))
    return FD_ERR_INVALID_ARG;
  if (epilogue < FD_EPI_F32 || epilogue > FD_EPI_SWIGLU) return FD_ERR_INVALID_ARG;
  if (epilogue == FD_EPI_GELU && N % 64) return FD_ERR_INVALID_ARG;
  if (epilogue == FD_EPI_SWIGLU && N % 128) return FD_ERR_INVALID_ARG;
  const bool bf16_out = epilogue == FD_EPI_GELU || epilogue == FD_EPI_SWIGLU;
  const int epi = epilogue == FD_EPI_SWIGLU ? fd::EPI_SWIGLU : epilogue;
  const int step = epilogue == FD_EPI_SWIGLU ? 128 : bf16_out ? 64 : 32;
  if (bn == 0) {
    const TileChoice t = pick_tile(M, N, K, step, false, pair);
    bn = t.bn;
    pair = t.pair ? 2 : 1;
  }
  if (pair == 0) pair = 1;
  if (!fd::gemm_bn_supported(bn) || !fd::gemm_bn_fits_epilogue(bn, epi) || (pair == 2 && bn < 96))
    return FD_ERR_INVALID_ARG;
  if (epilogue == FD_EPI_TUP && (tup_hidden < 32 || tup_hidden % 32 || N % tup_hidden))
    return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  CUtensorMap ta, tb;
  if (!tmap_bf16(&ta, A, K, M, static_cast<uint64_t>(K) * 2, 64, 128) ||
      !tmap_bf16(&tb, W, K, N, static_cast<uint64_t>(K) * 2, 64, pair == 2 ? bn / 2 : bn))
    return FD_ERR_CUDA;
  CUtensorMap to;
  bool ok;
  if (epilogue == FD_EPI_GELU) ok = tmap_out_bf16(&to, out, N, M, N);
  else if (epilogue == FD_EPI_SWIGLU) ok = tmap_out_bf16(&to, out, N / 2, M, N / 2);
  else if (epilogue == FD_EPI_TUP) ok = tmap_out_tup(&to, out, tup_hidden, M, N / tup_hidden);
  else ok = tmap_out_f32(&to, out, N, M, N);
  if (!ok) return FD_ERR_CUDA;
  fd::GemmParams p{};
  p.M = M; p.N = N; p.K = K; p.epi = epi; p.bias = bias; p.err = err_dev;
  if (bf16_out) {
    p.out_bf16 = static_cast<__nv_bfloat16*>(out);
  } else {
    p.out_f32 = static_cast<float*>(out);
  }
  p.ld_out = epilogue == FD_EPI_SWIGLU ? N / 2 : N;
  p.tup_tokens = M;
  p.tup_hidden = tup_hidden;
  return launch_ok(fd::launch_gemm(ta, tb, to, to, to, p, bn, pair == 2, num_sms(),
                                   static_cast<cudaStream_t>(stream)));
}

fd_status fd_op_linear_pixel(int M, int K, const void* A, const void* W, const float* bias,
                             int frames, int grid_h, int grid_w, int channels, int rs,
                             int out_dtype, void* pixels, int* err_dev, void* stream) {
  if (A == nullptr || W == nullptr || bias == nullptr || pixels == nullptr ||
      err_dev == nullptr || M < 1 || K < 1 || grid_h < 1 || grid_w < 1 || channels < 1 ||
      frames < 1 || (out_dtype != FD_DTYPE_F32 && out_dtype != FD_DTYPE_U8))
    return FD_ERR_INVALID_ARG;
  if (!fd::gemm_pixel_epilogue_ok(256, false, rs) || K % 8) return FD_ERR_INVALID_ARG;
  const long long L = static_cast<long long>(grid_h) * grid_w;
  const long long N = static_cast<long long>(channels) * rs * rs;
  if (N % 32 || N > (1 << 20) || L * frames > M || L > (1 << 24)) return FD_ERR_INVALID_ARG;
  if (!aligned16(A) || !aligned16(W) || !aligned16(bias) || !aligned16(pixels))
    return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  CUtensorMap ta, tb;
  if (!tmap_bf16(&ta, A, K, M, static_cast<uint64_t>(K) * 2, 64, 128) ||
      !tmap_bf16(&tb, W, K, static_cast<int>(N), static_cast<uint64_t>(K) * 2, 64, 256))
    return FD_ERR_CUDA;
  fd::GemmParams p{};
  p.M = M; p.N = static_cast<int>(N); p.K = K; p.epi = fd::EPI_PIXEL; p.bias = bias;
  p.err = err_dev;
  p.pix = {pixels, out_dtype == FD_DTYPE_U8 ? 1 : 0, frames, static_cast<int>(L), grid_h, grid_w,
           rs};
  return launch_ok(fd::launch_gemm(ta, tb, ta, ta, ta, p, 256, false, num_sms(),
                                   static_cast<cudaStream_t>(stream)));
}

fd_status fd_op_qkv(int M, int K, const void* A, const void* Wqkv, const float* bqkv,
                    const float* knorm_g, const float* norm2_g, int qk_norm, int heads,
                    int groups, int tokens, int grid_w, int frames_per_chunk, int window, int t,
                    float eps, float rope_base, const float* rope_t, void* q_out, void* k_ring,
                    void* vt_ring, int ring_pitch, int bn, int* err_dev, void* stream) {
  if (!A || !Wqkv || !bqkv || !knorm_g || !norm2_g || !q_out || !k_ring || !vt_ring ||
      !err_dev || !rope_t || (qk_norm != 0 && qk_norm != 1))
    return FD_ERR_INVALID_ARG;
  if (heads < 1 || groups < 1 || heads % groups || tokens < 1 || grid_w < 1 ||
      tokens % grid_w || frames_per_chunk < 1 || window < 1 || t < 0 || K < 8 || K % 8)
    return FD_ERR_INVALID_ARG;
  if (M != frames_per_chunk * tokens) return FD_ERR_INVALID_ARG;
  if (ring_pitch < window * M || ring_pitch % 128) return FD_ERR_INVALID_ARG;
  if (!aligned16(q_out) || !aligned16(k_ring) || !aligned16(vt_ring) || !aligned16(bqkv))
    return FD_ERR_INVALID_ARG;
  const int N = (heads + 2 * groups) * kHeadDim;
  bool pair = false;  // an explicit width runs on single CTAs; 0 = the launch-shape model
  if (bn == 0) {
    const TileChoice t = pick_tile(M, N, K, 64, false);
    bn = t.bn;
    pair = t.pair;
  }
  if (!fd::gemm_bn_supported(bn) || !fd::gemm_bn_fits_epilogue(bn, fd::EPI_QKV))
    return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  CUtensorMap ta, tb;
  if (!tmap_bf16(&ta, A, K, M, static_cast<uint64_t>(K) * 2, 64, 128) ||
      !tmap_bf16(&tb, Wqkv, K, N, static_cast<uint64_t>(K) * 2, 64, pair ? bn / 2 : bn))
    return FD_ERR_CUDA;
  fd::GemmParams p{};
  p.M = M; p.N = N; p.K = K; p.epi = fd::EPI_QKV; p.bias = bqkv; p.err = err_dev;
  fd::QkvEpi& q = p.qkv;
  q.heads = heads; q.groups = groups; q.knorm_g = knorm_g; q.vnorm_g = norm2_g;
  q.qk_norm = qk_norm;
  q.q_out = static_cast<__nv_bfloat16*>(q_out);
  q.k_ring = static_cast<__nv_bfloat16*>(k_ring);
  q.vt_ring = static_cast<__half*>(vt_ring);
  q.ring_pitch = ring_pitch; q.tokens = tokens; q.grid_w = grid_w;
  q.frames_per_chunk = frames_per_chunk; q.window = window; q.step_dev = nullptr;
  q.step_host = t; q.eps = eps;
  fill_rope(q, rope_base);
  q.rope_t = reinterpret_cast<const float2*>(rope_t);
  p.v_tma = M % 8 == 0 ? 1 : 0;
  CUtensorMap tq, tk, tv;
  if (!tmap_out_bf16(&tq, q_out, static_cast<uint64_t>(heads) * kHeadDim, M,
                     static_cast<uint64_t>(heads) * kHeadDim) ||
      !tmap_kring_store(&tk, k_ring, M, window, groups, ring_pitch))
    return FD_ERR_CUDA;
  if (p.v_tma) {
    if (!tmap_vring_store(&tv, vt_ring, M, window, groups, ring_pitch)) return FD_ERR_CUDA;
  } else {
    tv = tk;
  }
  return launch_ok(fd::launch_gemm(ta, tb, tq, tk, tv, p, bn, pair, num_sms(),
                                   static_cast<cudaStream_t>(stream)));
}

size_t fd_attention_workspace_bytes(int Lq, int heads, int groups, int n_keys, int parts) {
  if (Lq < 1 || heads < 1 || groups < 1 || heads % groups || n_keys < 1 || parts < 0 ||
      parts > kMaxAttnParts)
    return 0;
  if (parts == 0) parts = choose_parts(Lq, heads, groups, n_keys);
  return fd::attention_workspace_floats(parts, fd::attention_units(Lq, heads, groups)) * 4;
}

fd_status fd_op_attention(int Lq, int heads, int groups, const void* q, const void* k_ring,
                          const void* vt_ring, int ring_pitch, int n_keys, void* out,
                          int parts, void* workspace, int* err_dev, void* stream) {
  if (!q || !k_ring || !vt_ring || !out || !err_dev) return FD_ERR_INVALID_ARG;
  if (Lq < 1 || heads < 1 || groups < 1 || heads % groups || n_keys < 1 ||
      n_keys > ring_pitch || ring_pitch % 128 || parts < 0 || parts > kMaxAttnParts)
    return FD_ERR_INVALID_ARG;
  if (parts == 0) parts = choose_parts(Lq, heads, groups, n_keys);
  if (parts > 1 && (workspace == nullptr || !aligned16(workspace))) return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  const uint64_t NQ = static_cast<uint64_t>(heads) * kHeadDim;
  CUtensorMap tq, tq8, tk, tv;
  if (!tmap_bf16(&tq, q, NQ, Lq, NQ * 2, 64, 128) || !tmap_bf16(&tq8, q, NQ, Lq, NQ * 2, 64, 8) ||
      !tmap_bf16(&tk, k_ring, kHeadDim, static_cast<uint64_t>(groups) * ring_pitch, kHeadDim * 2,
                 64, 128) ||
      !tmap_f16(&tv, vt_ring, ring_pitch, static_cast<uint64_t>(groups) * kHeadDim,
                 static_cast<uint64_t>(ring_pitch) * 2, 64, 64))
    return FD_ERR_CUDA;
  fd::AttnParams a{};
  a.Lq = Lq; a.heads = heads; a.groups = groups; a.ring_pitch = ring_pitch;
  a.rows_per_chunk = n_keys; a.window = 1; a.step_dev = nullptr; a.n_keys_host = n_keys;
  a.out = static_cast<__nv_bfloat16*>(out); a.ld_out = static_cast<int>(NQ);
  a.scale_log2 = static_cast<float>(1.4426950408889634 / 8.0);
  a.err = err_dev;
  a.lq_pad = fd::attention_lq_pad(Lq);
  a.parts = parts;
  const int pairs = fd::attention_units(Lq, heads, groups);
  fd::attention_workspace_split(parts > 1 ? static_cast<float*>(workspace) : nullptr, parts,
                                pairs, a);
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the per-pair counters must start at zero (each launch leaves them at zero)
  if (a.counters != nullptr &&
      cudaMemsetAsync(a.counters, 0, sizeof(int) * pairs, s) !=
          cudaSuccess)
    return FD_ERR_CUDA;
  return launch_ok(fd::launch_attention(tq, tq8, tk, tv, a, s));
}

}  // extern "C"

// ---------------------------------------------------------------- allocation-free attention
// Workspace of fd_op_attention_static: the library's own static device memory, so that the
// call needs no allocation. Host code only uses its device address, looked up per CUDA context.
static __device__ __align__(256) float g_attn_static_scratch[FD_STATIC_ATTN_SCRATCH_BYTES / 4];

namespace {
std::mutex g_static_scratch_mu;
// (context id, device address) of the contexts seen so far. The array's address belongs to the
// context that loaded the module: after a device reset the primary context (and its id) is new,
// so the address is looked up again instead of reusing a stale one.
constexpr int kMaxContexts = 64;
unsigned long long g_static_ctx_id[kMaxContexts] = {};
float* g_static_ctx_addr[kMaxContexts] = {};
int g_static_ctx_n = 0;
PFN_cuCtxGetCurrent_v4000 g_ctx_current = nullptr;
PFN_cuCtxGetId_v12000 g_ctx_id = nullptr;

// id of the current CUDA context (0 if none or unavailable)
unsigned long long current_context_id() {
  if (g_ctx_current == nullptr || g_ctx_id == nullptr) {
    cudaDriverEntryPointQueryResult q;
    void* f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 4000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      g_ctx_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(f);
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      g_ctx_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(f);
    if (g_ctx_current == nullptr || g_ctx_id == nullptr) return 0;
  }
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (g_ctx_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
  if (g_ctx_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// device address of g_attn_static_scratch in the current context (looked up once per context,
// with that context current)
fd_status static_scratch_address(float** out) {
  std::lock_guard<std::mutex> lock(g_static_scratch_mu);
  unsigned long long id = current_context_id();
  for (int i = 0; id != 0 && i < g_static_ctx_n; ++i)
    if (g_static_ctx_id[i] == id) {
      *out = g_static_ctx_addr[i];
      return FD_OK;
    }
  if (g_static_ctx_n == kMaxContexts) return FD_ERR_UNSUPPORTED;
  // first call in this context: the lookup also makes the device's primary context current
  // on this thread if nothing had yet (no allocation either way)
  void* addr = nullptr;
  if (cudaGetSymbolAddress(&addr, g_attn_static_scratch) != cudaSuccess || addr == nullptr)
    return FD_ERR_CUDA;
  id = current_context_id();
  if (id == 0) return FD_ERR_CUDA;
  g_static_ctx_id[g_static_ctx_n] = id;
  g_static_ctx_addr[g_static_ctx_n] = static_cast<float*>(addr);
  ++g_static_ctx_n;
  *out = static_cast<float*>(addr);
  return FD_OK;
}
}  // namespace

extern "C" {

fd_status fd_op_attention_static(int Lq, int heads, int groups, const void* q,
                                 const void* k_ring, const void* vt_ring, int ring_pitch,
                                 int n_keys, void* out, int parts, int* err_dev, void* stream) {
  if (Lq < 1 || heads < 1 || groups < 1 || heads % groups || n_keys < 1 || parts < 0 ||
      parts > kMaxAttnParts)
    return FD_ERR_INVALID_ARG;
  if (parts == 0) parts = choose_parts(Lq, heads, groups, n_keys);
  if (fd::attention_workspace_floats(parts, fd::attention_units(Lq, heads, groups)) * 4 >
      FD_STATIC_ATTN_SCRATCH_BYTES)
    return FD_ERR_INVALID_ARG;
  float* ws = nullptr;
  if (parts > 1) {
    const fd_status st = static_scratch_address(&ws);
    if (st != FD_OK) return st;
  }
  return fd_op_attention(Lq, heads, groups, q, k_ring, vt_ring, ring_pitch, n_keys, out, parts,
                         ws, err_dev, stream);
}

fd_status fd_op_rope_table(int t, int frames_per_chunk, float rope_base, float* table,
                           void* stream) {
  if (t < 0 || frames_per_chunk < 1 || table == nullptr || !(rope_base > 1.f))
    return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  double inv[fd::kRopePairs];
  temporal_inv_freq(rope_base, inv);
  const int frames[1] = {frames_per_chunk};
  return launch_ok(fd::launch_rope_table(nullptr, t, 1, frames, rope_band_t(), inv,
                                         reinterpret_cast<float2*>(table),
                                         static_cast<cudaStream_t>(stream)));
}

fd_status fd_op_kv_append(const float* k, const float* v, int groups, int rows, int window,
                          int t, int ring_pitch, void* k_ring, void* vt_ring, void* stream) {
  if (!k || !v || !k_ring || !vt_ring || groups < 1 || rows < 1 || window < 1 || t < 0)
    return FD_ERR_INVALID_ARG;
  if (ring_pitch < window * rows) return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  return launch_ok(fd::launch_kv_append(k, v, groups, rows, t % window, ring_pitch,
                                        static_cast<__nv_bfloat16*>(k_ring),
                                        static_cast<__half*>(vt_ring),
                                        static_cast<cudaStream_t>(stream)));
}

fd_status fd_op_rmsnorm(const float* h, const float* g, int M, int D, float eps, void* u,
                        void* stream) {
  if (!h || !g || !u || M < 1 || D < 128 || D % 128 || !aligned16(h) || !aligned16(g))
    return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  return launch_ok(fd::launch_rmsnorm(h, g, M, D, eps, static_cast<__nv_bfloat16*>(u),
                                      static_cast<cudaStream_t>(stream)));
}

fd_status fd_op_rmsnorm_e4m3(const float* h, const float* g, int M, int D, float eps,
                             float out_scale, void* u, void* stream) {
  if (!h || !g || !u || M < 1 || D < 128 || D % 128 || !aligned16(h) || !aligned16(g) ||
      !aligned16(u) || !(out_scale > 0.f))
    return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  return launch_ok(fd::launch_rmsnorm_e4m3(h, g, M, D, eps, static_cast<uint8_t*>(u), out_scale,
                                           static_cast<cudaStream_t>(stream)));
}

fd_status fd_op_linear_e4m3(int epilogue, int M, int N, int K, const void* A, const void* W,
                            const float* col_scale, const float* bias, void* out,
                            float out_scale, int bn, int* err_dev, void* stream) {
  if (M < 1 || N < 1 || K < 16 || !A || !W || !col_scale || !bias || !out || !err_dev)
    return FD_ERR_INVALID_ARG;
  if (N % 32 || K % 16 || !aligned16(A) || !aligned16(W) || !aligned16(out) ||
      !aligned16(bias) || !aligned16(col_scale))
    return FD_ERR_INVALID_ARG;
  if (epilogue != FD_EPI_F32 && epilogue != FD_EPI_RESID && epilogue != FD_EPI_GELU &&
      epilogue != FD_EPI_SWIGLU)
    return FD_ERR_INVALID_ARG;
  const bool gated = epilogue == FD_EPI_SWIGLU;
  const bool f8_out = epilogue == FD_EPI_GELU || gated;
  if (f8_out && (N % (gated ? 256 : 128) || !(out_scale > 0.f))) return FD_ERR_INVALID_ARG;
  const int epi = gated ? fd::EPI_SWIGLU_F8 : f8_out ? fd::EPI_GELU_F8 : epilogue;
  if (bn == 0) bn = pick_bn_step(M, N, gated ? 256 : f8_out ? 128 : 32, f8_out);
  if (!fd::gemm_bn_supported(bn) || !fd::gemm_bn_fits_epilogue(bn, epi))
    return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  CUtensorMap ta, tb, to;
  if (!tmap_e4m3(&ta, A, K, M, K, 128) || !tmap_e4m3(&tb, W, K, N, K, bn)) return FD_ERR_CUDA;
  const int n_out = gated ? N / 2 : N;
  if (!(f8_out ? tmap_out_e4m3(&to, out, n_out, M, n_out) : tmap_out_f32(&to, out, N, M, N)))
    return FD_ERR_CUDA;
  fd::GemmParams p{};
  p.M = M; p.N = N; p.K = K; p.epi = epi; p.bias = bias; p.err = err_dev;
  p.fp8 = 1;
  p.col_scale = col_scale;
  p.out_scale = out_scale;
  if (f8_out) p.out_f8 = static_cast<uint8_t*>(out);
  else p.out_f32 = static_cast<float*>(out);
  p.ld_out = n_out;
  return launch_ok(fd::launch_gemm(ta, tb, to, to, to, p, bn, false, num_sms(),
                                   static_cast<cudaStream_t>(stream)));
}

fd_status fd_op_unshuffle(const float* z, int C, int H, int W, int p, void* x0, void* stream) {
  if (!z || !x0 || C < 1 || p < 1 || H < p || W < p || H % p || W % p) return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  return launch_ok(fd::launch_unshuffle(z, C, H, W, p, static_cast<__nv_bfloat16*>(x0),
                                        static_cast<cudaStream_t>(stream)));
}

fd_status fd_op_pixel_head(const float* F, int frames, int grid_h, int grid_w, int channels,
                           int rs, int out_dtype, void* pixels, void* stream) {
  if (!F || !pixels || frames < 1 || grid_h < 1 || grid_w < 1 || channels < 1 || rs < 4 ||
      rs % 4 || !aligned16(F) || !aligned16(pixels))
    return FD_ERR_INVALID_ARG;
  if (out_dtype != FD_DTYPE_F32 && out_dtype != FD_DTYPE_U8) return FD_ERR_INVALID_ARG;
  fd_status st = check_device();
  if (st) return st;
  return launch_ok(fd::launch_pixel_head(F, frames, grid_h, grid_w, channels, rs,
                                         out_dtype == FD_DTYPE_U8 ? 1 : 0, pixels,
                                         static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
