// Streaming training step on the GPU (Sec. 3.3 "Training--Inference Consistency", Sec. 3.5
// Eq. loss, its L1 term): the loss of a clip of T latent frames and the gradient of every
// decoder parameter.
//
// Training through the rolling cache has the gradient of one pass over the whole clip under
// the block sliding-window mask (query chunk i sees key chunks i-W < j <= i), so the GPU runs
// all T chunks at once: the forward of every block with its activations kept, the L1 term of
// the pixels, then the backward block by block in reverse. Every product runs on the tensor
// cores with bf16 operands and fp32 accumulation:
//   - the linear layers, their input gradients dX = dY W (with the transposed weights) and
//     weight gradients dW = dY^T X (with transposed activations): the library's GEMM
//     (gemm_view);
//   - the attention forward: the decode's batched attention kernel with one stream per query
//     chunk over the window of its key chunks, writing each row's log-sum-exp (attn_fwd);
//   - the attention backward per (query chunk, KV group): one launch for S = Q K^T and
//     dP = dO V^T with the softmax derivative dS = P (dP - rowsum(dO O)) in its epilogue
//     (scores_bwd: S and dP stay in tensor memory), then dQ = dS K, dK += dS^T Q, dV += P^T dO
//     on the GEMM (attn_bwd).
// Row-wise and element-wise steps (RMSNorm and its backward, KV-norm / QK-norm with 3D-RoPE and
// their backward, GELU and GELU', rowsum(dO O), the L1 term through the pixel shuffle, bias and
// gain sums) are the kernels below. Where a stack's keys per chunk are not a multiple of 8, its
// attention forward is materialised instead (S, the band softmax, O = P V).
//
// Rows: chunk c's L tokens sit at rows c Lp .. c Lp + L - 1 with Lp = 128 ceil(L / 128), the
// refined frame (c, tau) at rows (c r_t + tau) Lp ...; padding rows carry finite values
// forward (they are never keys: the softmax masks them) and exactly zero gradient backward, so
// they add nothing to any weight gradient.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>
#include <vector>

#include "fd_internal.h"
#include "flashdec.h"

namespace fd {
namespace train {

using bf16 = __nv_bfloat16;
constexpr int kDh = kHeadDim;
constexpr int kBandS = kHeadDim / 6;                  // pairs per spatial band (10)
constexpr int kBandT = kHeadDim / 2 - 2 * kBandS;     // temporal pairs (12)

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__global__ void to_bf16_kernel(const float* __restrict__ x, long long n, bf16* __restrict__ y) {
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x)
    y[i] = __float2bfloat16_rn(x[i]);
}

// y[c][r] = x[r][c] for a rows x cols block (pitches in elements), through a padded tile
template <typename T>
__global__ void transpose_kernel(const T* __restrict__ x, int rows, int cols, int ldx,
                                 T* __restrict__ y, int ldy) {
  __shared__ T tile[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = r0 + i, c = c0 + threadIdx.x;
    if (r < rows && c < cols) tile[i][threadIdx.x] = x[static_cast<size_t>(r) * ldx + c];
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int c = c0 + i, r = r0 + threadIdx.x;
    if (r < rows && c < cols) y[static_cast<size_t>(c) * ldy + r] = tile[threadIdx.x][i];
  }
}

// GELU, exact (erf) form, and its derivative Phi(z) + z phi(z)
__global__ void gelu_fwd_kernel(const float* __restrict__ z, long long n, bf16* __restrict__ a) {
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const float v = z[i];
    a[i] = __float2bfloat16_rn(0.5f * v * (1.0f + erff(v * 0.70710678118654752f)));
  }
}
__global__ void gelu_bwd_kernel(const float* __restrict__ z, const float* __restrict__ da,
                                long long n, float* __restrict__ dz, bf16* __restrict__ dz16) {
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const float v = z[i];
    const float Phi = 0.5f * (1.0f + erff(v * 0.70710678118654752f));
    const float phi = 0.39894228040143268f * expf(-0.5f * v * v);
    const float g = da[i] * (Phi + v * phi);
    dz[i] = g;
    dz16[i] = __float2bfloat16_rn(g);
  }
}

// RMSNorm backward, one warp per row (y = x r g, r = (mean(x^2) + eps)^(-1/2), n = D):
// dx = r (dy g) - x r^3 sum_j(dy_j g_j x_j) / n (+ add), t = dy x r (the gain's gradient
// summed over rows)
__global__ void rmsnorm_bwd_kernel(const float* __restrict__ x, const float* __restrict__ g,
                                   const float* __restrict__ dy, const float* __restrict__ add,
                                   int M, int D, float eps, float* __restrict__ dx,
                                   float* __restrict__ t) {
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= M) return;
  const float* xr = x + static_cast<size_t>(row) * D;
  const float* dr = dy + static_cast<size_t>(row) * D;
  float ss = 0.f, se = 0.f;
  for (int j = lane; j < D; j += 32) {
    const float v = xr[j];
    ss = fmaf(v, v, ss);
    se = fmaf(dr[j] * g[j], v, se);
  }
  ss = warp_sum(ss);
  se = warp_sum(se);
  const float r = rsqrtf(ss / D + eps);
  const float c = r * r * r * se / D;
  for (int j = lane; j < D; j += 32) {
    const size_t k = static_cast<size_t>(row) * D + j;
    float v = r * dr[j] * g[j] - xr[j] * c;
    if (add != nullptr) v += add[k];
    dx[k] = v;
    t[k] = dr[j] * xr[j] * r;
  }
}

// Gated MLP (the XL layout, reading R7): layer 1's output z [M][2 Dm] holds, on the device,
// the gate and up columns of 32 hidden units side by side in blocks of 64 (gate unit 32 j + i
// at column 64 j + i, its up column at 64 j + 32 + i); a = SiLU(gate) up, in unit order.
__device__ __forceinline__ float logistic(float x) { return 1.0f / (1.0f + expf(-x)); }
__global__ void swiglu_fwd_kernel(const float* __restrict__ z, long long M, int Dm,
                                  bf16* __restrict__ a) {
  const long long n = M * Dm;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long m = i / Dm;
    const int u = static_cast<int>(i % Dm);
    const float* zr = z + m * 2 * Dm + (u / 32) * 64 + u % 32;
    const float g = zr[0], up = zr[32];
    a[i] = __float2bfloat16_rn(g * logistic(g) * up);
  }
}
// its backward: d gate = da up SiLU'(gate) with SiLU'(x) = s(x) (1 + x (1 - s(x))), d up =
// da SiLU(gate); dz in the interleaved layout, fp32 and a bf16 copy
__global__ void swiglu_bwd_kernel(const float* __restrict__ z, const float* __restrict__ da,
                                  long long M, int Dm, float* __restrict__ dz,
                                  bf16* __restrict__ dz16) {
  const long long n = M * Dm;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long m = i / Dm;
    const int u = static_cast<int>(i % Dm);
    const long long c = m * 2 * Dm + (u / 32) * 64 + u % 32;
    const float g = z[c], up = z[c + 32], d = da[i];
    const float sg = logistic(g);
    const float dg = d * up * sg * (1.0f + g * (1.0f - sg)), du = d * g * sg;
    dz[c] = dg;
    dz[c + 32] = du;
    dz16[c] = __float2bfloat16_rn(dg);
    dz16[c + 32] = __float2bfloat16_rn(du);
  }
}
// rows of a gated layer 1's gradient from the device's interleaved order back to the blob's
// (gate rows, then up rows): dst row r = src row of blob row r
__global__ void gated_rows_kernel(const float* __restrict__ src, int rows, int len,
                                  float* __restrict__ dst) {
  const long long n = static_cast<long long>(rows) * len;
  const int gate = rows / 2;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int r = static_cast<int>(i / len), k = static_cast<int>(i % len);
    const int u = r < gate ? r : r - gate;
    const int dr = (u / 32) * 64 + (r < gate ? 0 : 32) + u % 32;
    dst[i] = src[static_cast<size_t>(dr) * len + k];
  }
}

// out[c] = sum over rows of x[r][c], rows in order (deterministic)
__global__ void colsum_kernel(const float* __restrict__ x, long long rows, int cols, int ld,
                              float* __restrict__ out) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= cols) return;
  float s = 0.f;
  for (long long r = 0; r < rows; ++r) s += x[r * ld + c];
  out[c] = s;
}

// The same sums in two stages, for many rows: part[k][c] = the sum of rows k R .. k R + R - 1
// (in order), then out[c] = the sum of the parts in order. A fixed order, so repeatable bits.
constexpr int kColsumRows = 256;
__global__ void colsum_part_kernel(const float* __restrict__ x, long long rows, int cols, int ld,
                                   float* __restrict__ part) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= cols) return;
  const long long r0 = static_cast<long long>(blockIdx.y) * kColsumRows;
  const long long r1 = r0 + kColsumRows < rows ? r0 + kColsumRows : rows;
  float s = 0.f;
  for (long long r = r0; r < r1; ++r) s += x[r * ld + c];
  part[static_cast<size_t>(blockIdx.y) * cols + c] = s;
}
__global__ void colsum_finish_kernel(const float* __restrict__ part, int parts, int cols,
                                     float* __restrict__ out) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= cols) return;
  float s = 0.f;
  for (int k = 0; k < parts; ++k) s += part[static_cast<size_t>(k) * cols + c];
  out[c] = s;
}

// RoPE tables (host-computed in double): temporal (cos, sin) [frames][kBandT], row and column
// [grid][kBandS]
struct Rope {
  const float2 *t, *y, *x;
};

// angle of pair i for frame f, grid row gy, column gx
__device__ __forceinline__ float2 rope_cs(const Rope& rp, int i, int f, int gy, int gx) {
  if (i < kBandT) return rp.t[f * kBandT + i];
  if (i < kBandT + kBandS) return rp.y[gy * kBandS + i - kBandT];
  return rp.x[gx * kBandS + i - kBandT - kBandS];
}

// RMS over the 64 values of one head with gain g
__device__ __forceinline__ void head_rms(float (&v)[kDh], const float* g, float eps) {
  float ss = 0.f;
#pragma unroll
  for (int j = 0; j < kDh; ++j) ss = fmaf(v[j], v[j], ss);
  const float r = rsqrtf(ss / kDh + eps);
#pragma unroll
  for (int j = 0; j < kDh; ++j) v[j] = v[j] * r * g[j];
}

// QKV forward of every row: slot < N query heads, then G key groups, then G value groups.
// q2 = RoPE(q0) (RMS with g2 first when qk_norm), k2 = RoPE(RMS(k0; gk)), v1 = RMS(v0; g2)
// (v0 when qk_norm). Outputs: q2 bf16 head-major per chunk of Pc rows, [M / Pc][N][Pc][64]
// (the rows of one chunk's heads of a KV group are then contiguous), k2 / v1 bf16 [G][M][64].
// With qr non-null, also: q rows bf16 [M][N 64] (the attention kernel's layout), and the
// real tokens' K bf16 [G][pitch][64] and V^T fp16 [G][64][pitch] without the padding rows
// (chunk c's Lu = Pc / Lp * L keys at c Lu ...), the keys of the fused band attention.
__global__ void qkv_fwd_kernel(const float* __restrict__ qkv, int M, int Pc, int Lp, int L,
                               int gw, int N, int G, int qk_norm, const float* __restrict__ gk,
                               const float* __restrict__ g2, float eps, Rope rp,
                               bf16* __restrict__ q2, bf16* __restrict__ k2,
                               bf16* __restrict__ v1, bf16* __restrict__ qr,
                               bf16* __restrict__ ku, __half* __restrict__ vtu, int pitch) {
  const int slots = N + 2 * G;
  const long long idx = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
  if (idx >= static_cast<long long>(M) * slots) return;
  const int row = static_cast<int>(idx / slots), slot = static_cast<int>(idx % slots);
  const int f = row / Lp, l = min(row % Lp, L - 1);  // padding rows take a real token's angles
  const int gy = l / gw, gx = l % gw;
  float v[kDh];
  const float* src = qkv + static_cast<size_t>(row) * slots * kDh + slot * kDh;
#pragma unroll
  for (int j = 0; j < kDh; ++j) v[j] = src[j];
  const bool is_q = slot < N, is_k = !is_q && slot < N + G;
  if (is_k) head_rms(v, gk, eps);
  else if (is_q ? qk_norm != 0 : qk_norm == 0) head_rms(v, g2, eps);
  bf16* dst;
  if (is_q) dst = q2 + (static_cast<size_t>(row / Pc * N + slot) * Pc + row % Pc) * kDh;
  else if (is_k) dst = k2 + (static_cast<size_t>(slot - N) * M + row) * kDh;
  else dst = v1 + (static_cast<size_t>(slot - N - G) * M + row) * kDh;
  if (is_q || is_k) {
#pragma unroll
    for (int i = 0; i < kDh / 2; ++i) {
      const float2 cs = rope_cs(rp, i, f, gy, gx);
      const float a = v[2 * i], b = v[2 * i + 1];
      v[2 * i] = a * cs.x - b * cs.y;
      v[2 * i + 1] = a * cs.y + b * cs.x;
    }
  }
#pragma unroll
  for (int j = 0; j < kDh; ++j) dst[j] = __float2bfloat16_rn(v[j]);
  if (qr == nullptr) return;
  if (is_q) {
    bf16* d = qr + static_cast<size_t>(row) * N * kDh + slot * kDh;
#pragma unroll
    for (int j = 0; j < kDh; ++j) d[j] = __float2bfloat16_rn(v[j]);
    return;
  }
  if (row % Lp >= L) return;  // padding rows are no keys
  const int key = row / Pc * (Pc / Lp * L) + row % Pc / Lp * L + row % Lp;
  if (is_k) {
    bf16* d = ku + (static_cast<size_t>(slot - N) * pitch + key) * kDh;
#pragma unroll
    for (int j = 0; j < kDh; ++j) d[j] = __float2bfloat16_rn(v[j]);
  } else {
    __half* d = vtu + static_cast<size_t>(slot - N - G) * kDh * pitch + key;
#pragma unroll
    for (int j = 0; j < kDh; ++j) d[static_cast<size_t>(j) * pitch] = __float2half_rn(v[j]);
  }
}

// RMS over one head, backward: x the pre-norm values, dy the gradient of the normed output
// (overwritten by dx); t = dy x r (gain's gradient term)
__device__ __forceinline__ void head_rms_bwd(const float (&x)[kDh], float (&dy)[kDh],
                                             const float* g, float eps, float* t) {
  float ss = 0.f, se = 0.f;
#pragma unroll
  for (int j = 0; j < kDh; ++j) {
    ss = fmaf(x[j], x[j], ss);
    se = fmaf(dy[j] * g[j], x[j], se);
  }
  const float r = rsqrtf(ss / kDh + eps);
  const float c = r * r * r * se / kDh;
#pragma unroll
  for (int j = 0; j < kDh; ++j) {
    t[j] = dy[j] * x[j] * r;
    dy[j] = r * dy[j] * g[j] - x[j] * c;
  }
}

// QKV backward of every row: dq2 fp32 [M / Pc][N][Pc][64] (the layout of q2), dk2 / dv1 fp32
// [G][M][64] -> dqkv fp32
// [M][(N + 2G) 64] (inverse RoPE: the rotation by the negated angle; then the per-head RMS
// backward where the forward normalised); gain terms tq [M N][64] (qk_norm), tk / tv [M G][64]
__global__ void qkv_bwd_kernel(const float* __restrict__ qkv, const float* __restrict__ dq2,
                               const float* __restrict__ dk2, const float* __restrict__ dv1,
                               int M, int Pc, int Lp, int L, int gw, int N, int G, int qk_norm,
                               const float* __restrict__ gk, const float* __restrict__ g2,
                               float eps, Rope rp, float* __restrict__ dqkv,
                               float* __restrict__ tq, float* __restrict__ tk,
                               float* __restrict__ tv) {
  const int slots = N + 2 * G;
  const long long idx = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
  if (idx >= static_cast<long long>(M) * slots) return;
  const int row = static_cast<int>(idx / slots), slot = static_cast<int>(idx % slots);
  const int f = row / Lp, l = min(row % Lp, L - 1);  // padding rows take a real token's angles
  const int gy = l / gw, gx = l % gw;
  const bool is_q = slot < N, is_k = !is_q && slot < N + G;
  float d[kDh], x[kDh];
  const float* src;
  if (is_q) src = dq2 + (static_cast<size_t>(row / Pc * N + slot) * Pc + row % Pc) * kDh;
  else if (is_k) src = dk2 + (static_cast<size_t>(slot - N) * M + row) * kDh;
  else src = dv1 + (static_cast<size_t>(slot - N - G) * M + row) * kDh;
#pragma unroll
  for (int j = 0; j < kDh; ++j) d[j] = src[j];
  if (is_q || is_k) {
#pragma unroll
    for (int i = 0; i < kDh / 2; ++i) {
      const float2 cs = rope_cs(rp, i, f, gy, gx);
      const float a = d[2 * i], b = d[2 * i + 1];
      d[2 * i] = a * cs.x + b * cs.y;
      d[2 * i + 1] = -a * cs.y + b * cs.x;
    }
  }
  const float* pre = qkv + static_cast<size_t>(row) * slots * kDh + slot * kDh;
#pragma unroll
  for (int j = 0; j < kDh; ++j) x[j] = pre[j];
  if (is_k) {
    head_rms_bwd(x, d, gk, eps, tk + (static_cast<size_t>(row) * G + slot - N) * kDh);
  } else if (is_q && qk_norm) {
    head_rms_bwd(x, d, g2, eps, tq + (static_cast<size_t>(row) * N + slot) * kDh);
  } else if (!is_q && !qk_norm) {
    head_rms_bwd(x, d, g2, eps, tv + (static_cast<size_t>(row) * G + slot - N - G) * kDh);
  }
  float* dst = dqkv + static_cast<size_t>(row) * slots * kDh + slot * kDh;
#pragma unroll
  for (int j = 0; j < kDh; ++j) dst[j] = d[j];
}

// Band softmax of one (query chunk, KV group): S fp32 [rows][n] (row pitch n), rows = the
// group's heads x the chunk's rows; column c is a key of a token (c mod Lp < L). P = softmax(S
// scale) over the valid columns (0 elsewhere) as bf16, and lse = log sum exp(S scale) of each
// row (natural log) for the backward. One warp per row: an online max / sum pass, then the
// write pass.
__global__ void softmax_lse_kernel(const float* __restrict__ S, int rows, int n, float scale,
                                   int Lp, int L, bf16* __restrict__ P16,
                                   float* __restrict__ lse) {
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const float* s = S + static_cast<size_t>(row) * n;
  float m = -INFINITY, sum = 0.f;
  for (int c = lane; c < n; c += 32) {
    if (c % Lp >= L) continue;
    const float v = s[c] * scale;
    if (v > m) {
      sum = sum * expf(m - v) + 1.0f;
      m = v;
    } else {
      sum += expf(v - m);
    }
  }
  const float mw = warp_max(m);
  sum = warp_sum(m == -INFINITY ? 0.f : sum * expf(m - mw));
  const float l = mw + logf(sum);
  for (int c = lane; c < n; c += 32) {
    const float p = c % Lp < L ? expf(s[c] * scale - l) : 0.f;
    P16[static_cast<size_t>(row) * n + c] = __float2bfloat16_rn(p);
  }
  if (lane == 0) lse[row] = l;
}

// delta[(c N + h) Pc + l] = sum_j dO[c Pc + l][h 64 + j] O[c Pc + l][h 64 + j]: dO fp32 and
// O bf16, both rows [M][N 64]; one warp per (chunk, head, row)
__global__ void delta_kernel(const float* __restrict__ dO, const bf16* __restrict__ O, int M,
                             int Pc, int N, float* __restrict__ delta) {
  const long long w = (blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= static_cast<long long>(M) * N) return;
  const int c = static_cast<int>(w / (static_cast<long long>(N) * Pc));
  const int h = static_cast<int>(w / Pc % N), l = static_cast<int>(w % Pc);
  const size_t e = (static_cast<size_t>(c) * Pc + l) * N * kDh + h * kDh;
  const float* a = dO + e;
  const bf16* b = O + e;
  float v = a[lane] * __bfloat162float(b[lane]) + a[lane + 32] * __bfloat162float(b[lane + 32]);
  v = warp_sum(v);
  if (lane == 0) delta[w] = v;
}

// head-major [M / Pc][N][Pc][64] fp32 <-> rows [M][N 64]: to_rows = 1 reads head-major x and
// writes bf16 rows; to_rows = 0 reads fp32 rows and writes bf16 head-major
__global__ void head_permute_kernel(const float* __restrict__ x, int M, int Pc, int N,
                                    int to_rows, bf16* __restrict__ y) {
  const long long total = static_cast<long long>(M) * N * kDh;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    // i indexes the rows layout: row m, head h, element j
    const long long m = i / (static_cast<long long>(N) * kDh);
    const int h = static_cast<int>(i / kDh % N), j = static_cast<int>(i % kDh);
    const long long hm = ((m / Pc * N + h) * Pc + m % Pc) * kDh + j;
    if (to_rows) y[i] = __float2bfloat16_rn(x[hm]);
    else y[hm] = __float2bfloat16_rn(x[i]);
  }
}

// L1 term of the pixels (reading T3: the mean of |x_hat - x| over the clip, unclamped output,
// reading T1) through the pixel shuffle: F [R][C rs^2] with refined row (c r_t + tau) Lp + l,
// target [T][C][r_t][H][W]; dF = sign(F - x) / total (0 on padding rows, and on chunk 0's
// frames tau >= first, which a one-frame first chunk does not emit); per-block partial sums of
// |F - x| into part[blockIdx.x] (fixed-order tree)
__global__ void l1_head_kernel(const float* __restrict__ F, const float* __restrict__ target,
                               int T, int rt, int first, int Lp, int L, int gh, int gw, int C,
                               int rs, float inv_total, float* __restrict__ dF,
                               float* __restrict__ part) {
  __shared__ float red[256];
  const int cols = C * rs * rs;
  const long long total = static_cast<long long>(T) * rt * Lp * cols;
  const long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
  float e = 0.f;
  if (i < total) {
    const long long row = i / cols;
    const int col = static_cast<int>(i % cols);
    const int l = static_cast<int>(row % Lp);
    const long long ft = row / Lp;  // c r_t + tau
    float g = 0.f;
    const int c = static_cast<int>(ft / rt), tau = static_cast<int>(ft % rt);
    if (l < L && (c > 0 || tau < first)) {
      const int ch = col / (rs * rs), ij = col % (rs * rs);
      const int ii = ij / rs, jj = ij % rs;
      const int h = l / gw, w = l % gw;
      const int H = gh * rs, W = gw * rs;
      const float x = target[((static_cast<size_t>(c) * C + ch) * rt + tau) * H * W +
                             static_cast<size_t>(h * rs + ii) * W + w * rs + jj];
      const float diff = F[i] - x;
      e = fabsf(diff);
      g = diff > 0.f ? inv_total : (diff < 0.f ? -inv_total : 0.f);
    }
    dF[i] = g;
  }
  red[threadIdx.x] = e;
  __syncthreads();
  for (int s = 128; s > 0; s >>= 1) {
    if (threadIdx.x < s) red[threadIdx.x] += red[threadIdx.x + s];
    __syncthreads();
  }
  if (threadIdx.x == 0) part[blockIdx.x] = red[0];
}

// one block of kLossThreads: thread t sums parts t, t + kLossThreads, ... in fp64, then a
// fixed-order tree over the threads (the same bits every step)
constexpr int kLossThreads = 1024;
__global__ void finish_loss_kernel(const float* __restrict__ part, int n, float inv_total,
                                   float* __restrict__ loss) {
  __shared__ double acc[kLossThreads];
  double s = 0.0;
  for (int i = threadIdx.x; i < n; i += kLossThreads) s += part[i];
  acc[threadIdx.x] = s;
  __syncthreads();
  for (int w = kLossThreads / 2; w > 0; w >>= 1) {
    if (static_cast<int>(threadIdx.x) < w) acc[threadIdx.x] += acc[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) *loss = static_cast<float>(acc[0] * inv_total);
}

// temporal upsampling layout (Eq. temporal_upsample, reading R6): channel block tau of token
// row c Lp + l of e [T Lp][r_t D] is refined row (c r_t + tau) Lp + l of hf [T r_t Lp][D]
__global__ void tup_permute_kernel(const float* __restrict__ src, int T, int rt, int Lp, int D,
                                   int inverse, float* __restrict__ dst, bf16* __restrict__ dst16) {
  const long long total = static_cast<long long>(T) * rt * Lp * D;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    // i indexes e: row c Lp + l, column tau D + d
    const long long erow = i / (static_cast<long long>(rt) * D);
    const int ecol = static_cast<int>(i % (static_cast<long long>(rt) * D));
    const int c = static_cast<int>(erow / Lp), l = static_cast<int>(erow % Lp);
    const int tau = ecol / D, d = ecol % D;
    const long long hrow = (static_cast<long long>(c) * rt + tau) * Lp + l;
    const long long h = hrow * D + d;
    if (inverse) {
      const float v = src[h];
      dst[i] = v;
      dst16[i] = __float2bfloat16_rn(v);
    } else {
      dst[h] = src[i];
    }
  }
}

}  // namespace train
}  // namespace fd

using fd::train::bf16;

// ---------------------------------------------------------------- the trainer object
struct fd_trainer_s {
  fd_config cfg;
  fd_weights w = nullptr;
  int T = 0;
  // shapes
  int C, H, W, p, D, N, G, NQ, QO, Dm, nb, nr, Wn, rt, rs, Cout, Cr, cin, gh, gw, L, Lp, MB, MR;
  int Dz = 0;          // MLP layer 1's outputs: Dm, or 2 Dm for the gated MLP (interleaved)
  bool gated = false;  // gated-SiLU MLP (the XL layout)
  bool f1 = false;     // chunk 0 emits one frame (first_chunk_frames = 1)
  float *dz32 = nullptr, *dwz = nullptr;  // gated: dz [M][2 Dm], layer 1's gradients (device order)
  float eps;
  std::vector<const void*> wt;   // device tensors of the weights, blob order
  std::vector<size_t> goff;      // element offset of each tensor in the gradient blob
  std::vector<void*> allocs;
  int* err = nullptr;
  float* zero_bias = nullptr;
  float2 *rope_t = nullptr, *rope_y = nullptr, *rope_x = nullptr;
  // transposed weights (bf16 [in][out]) of the linears used by the backward
  struct LinT {
    bf16 *qkv, *out, *mlp1, *mlp2;
  };
  std::vector<LinT> tB, tR;
  bf16 *t_tup = nullptr, *t_head1 = nullptr, *t_head2 = nullptr;
  // one stack's saved activations (per block) and its scratch
  struct Stack {
    int M, Pc;  // rows, rows per chunk
    std::vector<float*> h;  // block inputs (h[nblocks] = stack output), fp32 [M][D]
    std::vector<bf16*> u, q2, k2, v1, o, u2, a;
    std::vector<float*> qkv, hm, z, lse;  // lse [M / Pc][N][Pc]
    float* o32 = nullptr;  // head-major O of the materialised forward (scratch)
    // the fused band attention of the forward (the decode's batched attention kernel, one
    // stream per query chunk); off when its maps cannot be made
    struct {
      bool on = false;
      bf16* qr = nullptr;      // q rows [M][N 64]
      bf16* k = nullptr;       // K [G][pitch][64] of the real tokens
      __half* vt = nullptr;    // V^T [G][64][pitch]
      int pitch = 0, Lu = 0, parts = 1, pairs = 0;
      fd::AttnStream* streams = nullptr;  // device [T]
      int* steps = nullptr;               // device [T] = 0 .. T-1
      float* ws = nullptr;                // [T][ws_stride] partial results and counters
      size_t ws_stride = 0;
      CUtensorMap tmQ, tmQ8;
    } band;
  } sB, sR;
  // scratch
  bf16 *x0, *y16, *yh16, *a1, *vT, *kT, *do16, *dS, *P16, *dST, *PT, *QT, *dOT, *dy16, *dyT,
      *xT, *dqkv16;
  float *e, *z1, *F, *dF, *loss_part, *S, *delta, *dq2, *dk2, *dv1, *dqkv, *tq, *tk,
      *tv, *gA, *gB, *gC, *tbuf, *gtmp;
  int loss_blocks = 0;
  int hs = 1;  // heads of one KV group per attention product (a divisor of N / G)
  float* colsum_part = nullptr;  // partial column sums
  size_t colsum_elems = 0;
  // per-kernel profile (fd_train_profile_enable): events around each launch, by kernel kind
  struct Rec {
    int kind;
    cudaEvent_t a, b;
  };
  bool prof = false;
  std::vector<cudaEvent_t> ev_free, ev_all;
  std::vector<Rec> rec;
  cudaEvent_t event() {
    if (!ev_free.empty()) {
      cudaEvent_t e = ev_free.back();
      ev_free.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    ev_all.push_back(e);
    return e;
  }
};

namespace {

template <typename T>
T* dalloc(fd_trainer_s* tr, size_t elems, bool& ok) {
  void* ptr = nullptr;
  if (!ok || cudaMalloc(&ptr, elems * sizeof(T) + 256) != cudaSuccess) {
    ok = false;
    return nullptr;
  }
  tr->allocs.push_back(ptr);
  if (cudaMemset(ptr, 0, elems * sizeof(T) + 256) != cudaSuccess) ok = false;
  return static_cast<T*>(ptr);
}

int blocks_for(long long n, int threads) {
  long long b = (n + threads - 1) / threads;
  return static_cast<int>(b < 1 ? 1 : (b > 65535 * 16 ? 65535 * 16 : b));
}

double rope_inv_freq(int i, double base) {
  using fd::train::kBandS;
  using fd::train::kBandT;
  int j, d;
  if (i < kBandT) { j = i; d = 2 * kBandT; }
  else if (i < kBandT + kBandS) { j = i - kBandT; d = 2 * kBandS; }
  else { j = i - kBandT - kBandS; d = 2 * kBandS; }
  return std::pow(base, -2.0 * j / d);
}

// the launches of one step, in order on one stream; any failure ends the step
struct Run {
  fd_trainer_s* tr;
  cudaStream_t s;
  bool ok = true;
  cudaEvent_t t0 = nullptr;  // start event of the launch being profiled
  int t_kind = 0;

  void check(cudaError_t e) {
    if (e != cudaSuccess) ok = false;
  }
  // bracket the next launch with profile events (when the profile is enabled)
  bool begin(int kind) {
    if (!ok) return false;
    if (tr->prof) {
      t0 = tr->event();
      t_kind = kind;
      if (t0 != nullptr) check(cudaEventRecord(t0, s));
    }
    return ok;
  }
  void end() {
    if (t0 == nullptr) return;
    cudaEvent_t t1 = tr->event();
    if (t1 != nullptr) {
      check(cudaEventRecord(t1, s));
      tr->rec.push_back({t_kind, t0, t1});
    } else {
      tr->ev_free.push_back(t0);
    }
    t0 = nullptr;
  }
  void gemm(int kind, int epi, int M, int N, int K, const bf16* A, int lda, const bf16* Wm,
            int ldw, const float* bias, float* out, int ldo) {
    if (!begin(kind)) return;
    check(fd::gemm_view(epi, M, N, K, A, lda, Wm, ldw, bias ? bias : tr->zero_bias, out, ldo,
                        tr->err, s));
    end();
  }
  void bf(const float* x, long long n, bf16* y) {
    if (!begin(FD_TK_POINTWISE)) return;
    fd::train::to_bf16_kernel<<<blocks_for(n, 256), 256, 0, s>>>(x, n, y);
    check(cudaGetLastError());
    end();
  }
  template <typename T>
  void transpose(const T* x, int rows, int cols, int ldx, T* y, int ldy) {
    if (!begin(FD_TK_TRANSPOSE)) return;
    dim3 grid((cols + 31) / 32, (rows + 31) / 32);
    fd::train::transpose_kernel<T><<<grid, dim3(32, 8), 0, s>>>(x, rows, cols, ldx, y, ldy);
    check(cudaGetLastError());
    end();
  }
  void colsum(const float* x, long long rows, int cols, int ld, float* out) {
    const int parts = static_cast<int>((rows + fd::train::kColsumRows - 1) /
                                       fd::train::kColsumRows);
    if (static_cast<size_t>(parts) * cols > tr->colsum_elems) {
      ok = false;
      return;
    }
    if (!begin(FD_TK_POINTWISE)) return;
    fd::train::colsum_part_kernel<<<dim3((cols + 127) / 128, parts), 128, 0, s>>>(
        x, rows, cols, ld, tr->colsum_part);
    check(cudaGetLastError());
    fd::train::colsum_finish_kernel<<<(cols + 127) / 128, 128, 0, s>>>(tr->colsum_part, parts,
                                                                      cols, out);
    check(cudaGetLastError());
    end();
  }
  void copy(float* dst, const float* src, size_t n) {
    if (!begin(FD_TK_POINTWISE)) return;
    check(cudaMemcpyAsync(dst, src, sizeof(float) * n, cudaMemcpyDeviceToDevice, s));
    end();
  }
  void zero(float* dst, size_t n) {
    if (!begin(FD_TK_POINTWISE)) return;
    check(cudaMemsetAsync(dst, 0, sizeof(float) * n, s));
    end();
  }
  void rmsnorm(const float* x, const float* g, int M, bf16* u) {
    if (!begin(FD_TK_NORM)) return;
    check(fd::launch_rmsnorm(x, g, M, tr->D, tr->eps, u, s));
    end();
  }
  // dx = RMSNorm backward (+ add), the gain's gradient into grad
  void rmsnorm_bwd(const float* x, const float* g, const float* dy, const float* add, int M,
                   float* dx, float* grad) {
    if (!begin(FD_TK_NORM)) return;
    fd::train::rmsnorm_bwd_kernel<<<(M + 7) / 8, 256, 0, s>>>(x, g, dy, add, M, tr->D, tr->eps,
                                                             dx, tr->tbuf);
    check(cudaGetLastError());
    end();
    colsum(tr->tbuf, M, tr->D, tr->D, grad);
  }
  // weight gradient of a linear out = X W^T: dW [n_out][n_in] = dY^T X with dY16 [M][n_out]
  // and X16 [M][n_in] (bf16; K of the product = M rows, padding rows of dY are zero)
  void wgrad(const bf16* dY16, int n_out, const bf16* X16, int n_in, int M, float* dW) {
    bf16* dyT = tr->dyT;
    bf16* xT = tr->xT;
    transpose(dY16, M, n_out, n_out, dyT, M);
    transpose(X16, M, n_in, n_in, xT, M);
    if (n_in % 32 == 0) {
      gemm(FD_TK_WGRAD, fd::EPI_F32, n_out, n_in, M, dyT, M, xT, M, nullptr, dW, n_in);
    } else {  // the product in the other orientation (its N = n_out), then transposed
      gemm(FD_TK_WGRAD, fd::EPI_F32, n_in, n_out, M, xT, M, dyT, M, nullptr, tr->gtmp, n_out);
      transpose(tr->gtmp, n_in, n_out, n_out, dW, n_in);
    }
  }
  float* grad(float* g, size_t entry) { return g + tr->goff[entry]; }
  const float* wf(size_t entry) { return static_cast<const float*>(tr->wt[entry]); }
  const bf16* wb(size_t entry) { return static_cast<const bf16*>(tr->wt[entry]); }
};

// blob entries of block b of a stack starting at entry e0: norm1.g, qkv.w, qkv.b, knorm.g,
// (vnorm|qnorm).g, out.w, out.b, norm2.g, mlp1.w, mlp1.b, mlp2.w, mlp2.b
enum { kN1 = 0, kQW, kQB, kKG, kG2, kOW, kOB, kN2, kM1W, kM1B, kM2W, kM2B, kBlockEntries };

// attention forward of one block (Sec. 3.3, Eq. attention over the chunk window): O rows (bf16)
// into st.o and each row's log-sum-exp into st.lse. On the batched attention kernel when the
// stack's band maps exist; else materialised per (query chunk i, KV group g): the rows of the
// group's heads form one product with the window's keys (chunks max(0, i - W + 1) .. i,
// contiguous in k2 / v1): S = Q K^T, band softmax (P bf16 and the log-sum-exp), O = P V (head-
// major fp32 in st.o32, then permuted into st.o). A group's heads go tr->hs at a time (all of
// them unless S would pass its size bound).
void attn_fwd(Run& r, fd_trainer_s::Stack& st, int b) {
  fd_trainer_s* tr = r.tr;
  const int M = st.M, Pc = st.Pc, N = tr->N, hpg = N / tr->G, rows = tr->hs * Pc;
  if (st.band.on) {
    // the decode's batched attention kernel, one stream per query chunk: stream i's queries are
    // its Pc rows (padding rows computed, not used), its keys the window's real tokens; O as
    // bf16 rows into st.o, each row's log-sum-exp into st.lse
    auto& bd = st.band;
    fd::AttnParams a{};
    a.Lq = Pc; a.heads = N; a.groups = tr->G; a.ring_pitch = bd.pitch;
    a.rows_per_chunk = bd.Lu; a.window = tr->Wn; a.step_dev = bd.steps; a.n_keys_host = 0;
    a.out = st.o[b]; a.ld_out = tr->NQ;
    a.scale_log2 = static_cast<float>(1.4426950408889634 / 8.0);
    a.err = tr->err;
    a.lq_pad = fd::attention_lq_pad(Pc);
    a.parts = bd.parts;
    fd::attention_workspace_split(bd.ws, bd.parts, bd.pairs, a);
    a.streams = bd.streams; a.n_streams = tr->T; a.q_rows_stream = Pc;
    a.ws_stride = bd.ws_stride;
    a.lse = st.lse[b]; a.lse_pitch = Pc;
    if (r.begin(FD_TK_ATTN_GEMM)) {
      r.check(fd::launch_attention(bd.tmQ, bd.tmQ8, bd.tmQ, bd.tmQ, a, r.s));
      r.end();
    }
    return;
  }
  // V^T [G][64][M] for the P V products
  for (int g = 0; g < tr->G; ++g)
    r.transpose(st.v1[b] + static_cast<size_t>(g) * M * 64, M, 64, 64,
                tr->vT + static_cast<size_t>(g) * 64 * M, M);
  for (int i = 0; i < tr->T; ++i) {
    const int j0 = i - tr->Wn + 1 > 0 ? i - tr->Wn + 1 : 0;
    const int k0 = j0 * Pc, nk = (i + 1) * Pc - k0;
    for (int h0 = 0; h0 < N; h0 += tr->hs) {  // tr->hs heads of group h0 / hpg at a time
      const int g = h0 / hpg;
      const size_t q0 = (static_cast<size_t>(i) * N + h0) * Pc;  // first row, head-major
      r.gemm(FD_TK_ATTN_GEMM, fd::EPI_F32, rows, nk, 64, st.q2[b] + q0 * 64, 64,
             st.k2[b] + (static_cast<size_t>(g) * M + k0) * 64, 64, nullptr, tr->S, nk);
      if (r.begin(FD_TK_SOFTMAX)) {
        fd::train::softmax_lse_kernel<<<(rows + 7) / 8, 256, 0, r.s>>>(
            tr->S, rows, nk, 0.125f, tr->Lp, tr->L, tr->P16, st.lse[b] + q0);
        r.check(cudaGetLastError());
        r.end();
      }
      r.gemm(FD_TK_ATTN_GEMM, fd::EPI_F32, rows, 64, nk, tr->P16, nk,
             tr->vT + static_cast<size_t>(g) * 64 * M + k0, M, nullptr, st.o32 + q0 * 64, 64);
    }
  }
  if (r.begin(FD_TK_POINTWISE)) {  // O rows (bf16) for the output projection
    const long long n = static_cast<long long>(M) * tr->NQ;
    fd::train::head_permute_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(st.o32, M, Pc, N, 1,
                                                                         st.o[b]);
    r.check(cudaGetLastError());
    r.end();
  }
}

// attention backward of one block: dq2 (fp32, the head-major layout of q2), dk2, dv1 (fp32
// [G][M][64], accumulated over the query chunks whose windows hold each key; the group's heads
// sum inside each product) from dO (tr->gA, fp32 rows [M][N 64])
void attn_bwd(Run& r, fd_trainer_s::Stack& st, int b) {
  fd_trainer_s* tr = r.tr;
  const int M = st.M, Pc = st.Pc, N = tr->N, hpg = N / tr->G, rows = tr->hs * Pc;
  r.zero(tr->dk2, static_cast<size_t>(tr->G) * M * 64);
  r.zero(tr->dv1, static_cast<size_t>(tr->G) * M * 64);
  for (int g = 0; g < tr->G; ++g)
    r.transpose(st.k2[b] + static_cast<size_t>(g) * M * 64, M, 64, 64,
                tr->kT + static_cast<size_t>(g) * 64 * M, M);
  // dO head-major (bf16) and delta = rowsum(dO o O) of every (chunk, head, row)
  if (r.begin(FD_TK_POINTWISE)) {
    const long long n = static_cast<long long>(M) * tr->NQ;
    fd::train::head_permute_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(tr->gA, M, Pc, N, 0,
                                                                         tr->do16);
    r.check(cudaGetLastError());
    r.end();
  }
  if (r.begin(FD_TK_SOFTMAX)) {
    const long long n = static_cast<long long>(M) * N * 32;
    fd::train::delta_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(tr->gA, st.o[b], M, Pc, N,
                                                                  tr->delta);
    r.check(cudaGetLastError());
    r.end();
  }
  for (int i = 0; i < tr->T; ++i) {
    const int j0 = i - tr->Wn + 1 > 0 ? i - tr->Wn + 1 : 0;
    const int k0 = j0 * Pc, nk = (i + 1) * Pc - k0;
    for (int h0 = 0; h0 < N; h0 += tr->hs) {
      const int g = h0 / hpg;
      const size_t q0 = (static_cast<size_t>(i) * N + h0) * Pc;
      const bf16* Kw = st.k2[b] + (static_cast<size_t>(g) * M + k0) * 64;
      const bf16* Vw = st.v1[b] + (static_cast<size_t>(g) * M + k0) * 64;
      // S = Q K^T (recomputed) and dP = dO V^T in one launch, the softmax backward in its
      // epilogue: dS = P (dP - delta) / sqrt(D_h) with P = exp(S / sqrt(D_h) - lse), written as
      // dS, dS^T and P^T; S and dP are never stored
      if (r.begin(FD_TK_ATTN_GEMM)) {
        const fd::DsEpi ds{st.lse[b] + q0, tr->delta + q0, 0.125f, Pc, tr->Lp, tr->L,
                           tr->dS, tr->dST, tr->PT};
        r.check(fd::scores_bwd(rows, nk, st.q2[b] + q0 * 64, tr->do16 + q0 * 64, 64, Kw, Vw, 64,
                               ds, tr->err, r.s));
        r.end();
      }
      // dQ = dS K
      r.gemm(FD_TK_ATTN_GEMM, fd::EPI_F32, rows, 64, nk, tr->dS, nk,
             tr->kT + static_cast<size_t>(g) * 64 * M + k0, M, nullptr, tr->dq2 + q0 * 64, 64);
      // dK += dS^T Q, dV += P^T dO (K of both products: the group's rows)
      r.transpose(st.q2[b] + q0 * 64, rows, 64, 64, tr->QT, rows);
      r.gemm(FD_TK_ATTN_GEMM, fd::EPI_RESID, nk, 64, rows, tr->dST, rows, tr->QT, rows, nullptr,
             tr->dk2 + (static_cast<size_t>(g) * M + k0) * 64, 64);
      r.transpose(tr->do16 + q0 * 64, rows, 64, 64, tr->dOT, rows);
      r.gemm(FD_TK_ATTN_GEMM, fd::EPI_RESID, nk, 64, rows, tr->PT, rows, tr->dOT, rows, nullptr,
             tr->dv1 + (static_cast<size_t>(g) * M + k0) * 64, 64);
    }
  }
}

// one block forward (Sec. 3.2): st.h[b] -> st.h[b + 1], activations kept
void block_fwd(Run& r, fd_trainer_s::Stack& st, int b, size_t e0) {
  fd_trainer_s* tr = r.tr;
  const int M = st.M;
  r.rmsnorm(st.h[b], r.wf(e0 + kN1), M, st.u[b]);
  r.gemm(FD_TK_LINEAR, fd::EPI_F32, M, tr->QO, tr->D, st.u[b], tr->D, r.wb(e0 + kQW), tr->D, r.wf(e0 + kQB),
         st.qkv[b], tr->QO);
  if (r.begin(FD_TK_NORM)) {
    const fd::train::Rope rp{tr->rope_t, tr->rope_y, tr->rope_x};
    const long long n = static_cast<long long>(M) * (tr->N + 2 * tr->G);
    fd::train::qkv_fwd_kernel<<<blocks_for(n, 128), 128, 0, r.s>>>(
        st.qkv[b], M, st.Pc, tr->Lp, tr->L, tr->gw, tr->N, tr->G, tr->cfg.qk_norm, r.wf(e0 + kKG),
        r.wf(e0 + kG2), tr->eps, rp, st.q2[b], st.k2[b], st.v1[b], st.band.on ? st.band.qr : nullptr,
        st.band.k, st.band.vt, st.band.pitch);
    r.check(cudaGetLastError());
    r.end();
  }
  attn_fwd(r, st, b);
  r.copy(st.hm[b], st.h[b], static_cast<size_t>(M) * tr->D);
  r.gemm(FD_TK_LINEAR, fd::EPI_RESID, M, tr->D, tr->NQ, st.o[b], tr->NQ, r.wb(e0 + kOW), tr->NQ,
         r.wf(e0 + kOB), st.hm[b], tr->D);
  r.rmsnorm(st.hm[b], r.wf(e0 + kN2), M, st.u2[b]);
  r.gemm(FD_TK_LINEAR, fd::EPI_F32, M, tr->Dz, tr->D, st.u2[b], tr->D, r.wb(e0 + kM1W), tr->D,
         r.wf(e0 + kM1B), st.z[b], tr->Dz);
  if (r.begin(FD_TK_POINTWISE)) {
    const long long n = static_cast<long long>(M) * tr->Dm;
    if (tr->gated)
      fd::train::swiglu_fwd_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(st.z[b], M, tr->Dm,
                                                                         st.a[b]);
    else
      fd::train::gelu_fwd_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(st.z[b], n, st.a[b]);
    r.check(cudaGetLastError());
    r.end();
  }
  r.copy(st.h[b + 1], st.hm[b], static_cast<size_t>(M) * tr->D);
  r.gemm(FD_TK_LINEAR, fd::EPI_RESID, M, tr->D, tr->Dm, st.a[b], tr->Dm, r.wb(e0 + kM2W), tr->Dm,
         r.wf(e0 + kM2B), st.h[b + 1], tr->D);
}

// one block backward: dho (tr->gB, fp32 [M][D]) -> dh_in (tr->gB), gradients into g
void block_bwd(Run& r, fd_trainer_s::Stack& st, int b, size_t e0,
               const fd_trainer_s::LinT& lt, float* g) {
  fd_trainer_s* tr = r.tr;
  const int M = st.M, D = tr->D, Dm = tr->Dm, NQ = tr->NQ, QO = tr->QO;
  float* dho = tr->gB;
  r.bf(dho, static_cast<long long>(M) * D, tr->dy16);
  // MLP layer 2
  r.gemm(FD_TK_DGRAD, fd::EPI_F32, M, Dm, D, tr->dy16, D, lt.mlp2, D, nullptr, tr->gC, Dm);  // da
  r.wgrad(tr->dy16, D, st.a[b], Dm, M, r.grad(g, e0 + kM2W));
  r.colsum(dho, M, D, D, r.grad(g, e0 + kM2B));
  // GELU' (or the gated SiLU's derivative into the interleaved dz)
  const int Dz = tr->Dz;
  float* dz = tr->gated ? tr->dz32 : tr->gC;
  if (r.begin(FD_TK_POINTWISE)) {
    const long long n = static_cast<long long>(M) * Dm;
    if (tr->gated)
      fd::train::swiglu_bwd_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(st.z[b], tr->gC, M, Dm,
                                                                          dz, tr->dqkv16);
    else
      fd::train::gelu_bwd_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(st.z[b], tr->gC, n,
                                                                        tr->gC, tr->dqkv16);
    r.check(cudaGetLastError());
    r.end();
  }
  // MLP layer 1
  r.gemm(FD_TK_DGRAD, fd::EPI_F32, M, D, Dz, tr->dqkv16, Dz, lt.mlp1, Dz, nullptr, tr->gA, D);  // du2
  if (tr->gated) {  // gradients in the device's interleaved rows, then into the blob's order
    float* dwz = tr->dwz;
    float* dbz = tr->dwz + static_cast<size_t>(Dz) * D;
    r.wgrad(tr->dqkv16, Dz, st.u2[b], D, M, dwz);
    r.colsum(dz, M, Dz, Dz, dbz);
    if (r.begin(FD_TK_POINTWISE)) {
      const long long n = static_cast<long long>(Dz) * D;
      fd::train::gated_rows_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(
          dwz, Dz, D, r.grad(g, e0 + kM1W));
      r.check(cudaGetLastError());
      fd::train::gated_rows_kernel<<<blocks_for(Dz, 256), 256, 0, r.s>>>(
          dbz, Dz, 1, r.grad(g, e0 + kM1B));
      r.check(cudaGetLastError());
      r.end();
    }
  } else {
    r.wgrad(tr->dqkv16, Dz, st.u2[b], D, M, r.grad(g, e0 + kM1W));
    r.colsum(dz, M, Dz, Dz, r.grad(g, e0 + kM1B));
  }
  // RMSNorm 2, plus the residual
  r.rmsnorm_bwd(st.hm[b], r.wf(e0 + kN2), tr->gA, dho, M, tr->gC, r.grad(g, e0 + kN2));
  float* dhm = tr->gC;
  r.bf(dhm, static_cast<long long>(M) * D, tr->dy16);
  // output projection
  r.gemm(FD_TK_DGRAD, fd::EPI_F32, M, NQ, D, tr->dy16, D, lt.out, D, nullptr, tr->gA, NQ);  // dO (fp32)
  r.wgrad(tr->dy16, D, st.o[b], NQ, M, r.grad(g, e0 + kOW));
  r.colsum(dhm, M, D, D, r.grad(g, e0 + kOB));
  // attention (reads dO from gA)
  attn_bwd(r, st, b);
  // KV-norm / QK-norm and RoPE backward
  if (r.begin(FD_TK_NORM)) {
    const fd::train::Rope rp{tr->rope_t, tr->rope_y, tr->rope_x};
    const long long n = static_cast<long long>(M) * (tr->N + 2 * tr->G);
    fd::train::qkv_bwd_kernel<<<blocks_for(n, 128), 128, 0, r.s>>>(
        st.qkv[b], tr->dq2, tr->dk2, tr->dv1, M, st.Pc, tr->Lp, tr->L, tr->gw, tr->N, tr->G,
        tr->cfg.qk_norm, r.wf(e0 + kKG), r.wf(e0 + kG2), tr->eps, rp, tr->dqkv, tr->tq, tr->tk,
        tr->tv);
    r.check(cudaGetLastError());
    r.end();
  }
  r.colsum(tr->tk, static_cast<long long>(M) * tr->G, 64, 64, r.grad(g, e0 + kKG));
  if (tr->cfg.qk_norm)
    r.colsum(tr->tq, static_cast<long long>(M) * tr->N, 64, 64, r.grad(g, e0 + kG2));
  else
    r.colsum(tr->tv, static_cast<long long>(M) * tr->G, 64, 64, r.grad(g, e0 + kG2));
  r.bf(tr->dqkv, static_cast<long long>(M) * QO, tr->dqkv16);
  // QKV projection
  r.gemm(FD_TK_DGRAD, fd::EPI_F32, M, D, QO, tr->dqkv16, QO, lt.qkv, QO, nullptr, tr->gA, D);  // du
  r.wgrad(tr->dqkv16, QO, st.u[b], D, M, r.grad(g, e0 + kQW));
  r.colsum(tr->dqkv, M, QO, QO, r.grad(g, e0 + kQB));
  // RMSNorm 1, plus the residual: dh_in
  r.rmsnorm_bwd(st.h[b], r.wf(e0 + kN1), tr->gA, dhm, M, tr->gB, r.grad(g, e0 + kN1));
}

}  // namespace

extern "C" {

size_t fd_train_grad_elems(const fd_config* cfg) { return fd_weights_blob_elems(cfg); }

fd_status fd_train_create(const fd_config* cfg, fd_weights w, int chunks, fd_trainer* out) {
  if (out == nullptr || w == nullptr || cfg == nullptr) return FD_ERR_INVALID_ARG;
  *out = nullptr;
  const fd_config* wc = fd::weights_config(w);
  if (fd_weights_blob_elems(cfg) == 0 || std::memcmp(cfg, wc, sizeof(fd_config)) != 0)
    return FD_ERR_CONFIG;
  // the bf16-valued decoder: GELU or gated-SiLU MLPs, r_t frames per chunk or one from chunk 0
  if (cfg->mlp_fp8) return FD_ERR_CONFIG;
  if (chunks < 1 || chunks > 256) return FD_ERR_INVALID_ARG;
  fd_trainer tr = new (std::nothrow) fd_trainer_s;
  if (tr == nullptr) return FD_ERR_OOM;
  tr->cfg = *cfg;
  tr->w = w;
  tr->T = chunks;
  tr->C = cfg->latent_channels; tr->H = cfg->latent_h; tr->W = cfg->latent_w; tr->p = cfg->patch;
  tr->D = cfg->hidden; tr->N = cfg->heads; tr->G = cfg->kv_groups; tr->NQ = tr->N * 64;
  tr->QO = (tr->N + 2 * tr->G) * 64; tr->Dm = cfg->mlp_ratio * tr->D; tr->nb = cfg->n_blocks;
  tr->gated = cfg->mlp_gated != 0;
  tr->Dz = tr->gated ? 2 * tr->Dm : tr->Dm;
  tr->f1 = cfg->first_chunk_frames == 1;
  tr->nr = cfg->n_refine; tr->Wn = cfg->window; tr->rt = cfg->r_t;
  tr->rs = cfg->vae_spatial * cfg->patch; tr->Cout = cfg->out_channels;
  tr->Cr = tr->Cout * tr->rs * tr->rs; tr->cin = tr->C * tr->p * tr->p;
  tr->gh = tr->H / tr->p; tr->gw = tr->W / tr->p; tr->L = tr->gh * tr->gw;
  tr->Lp = (tr->L + 127) / 128 * 128;
  tr->MB = tr->T * tr->Lp;
  tr->MR = tr->T * tr->rt * tr->Lp;
  tr->eps = cfg->norm_eps;
  // tensors of the weights and their offsets in the gradient blob
  const size_t n_ent = fd::weights_entries(w, nullptr, 0);
  tr->wt.resize(n_ent);
  fd::weights_entries(w, tr->wt.data(), n_ent);
  {
    const size_t D = tr->D, blk[kBlockEntries] = {
        D, static_cast<size_t>(tr->QO) * D, static_cast<size_t>(tr->QO), 64, 64,
        D * tr->NQ, D, D, static_cast<size_t>(tr->Dz) * D, static_cast<size_t>(tr->Dz),
        D * tr->Dm, D};
    std::vector<size_t> elems = {D * tr->cin, D};
    for (int b = 0; b < tr->nb; ++b) elems.insert(elems.end(), blk, blk + kBlockEntries);
    elems.push_back(D);
    elems.push_back(static_cast<size_t>(tr->rt) * D * D);
    elems.push_back(static_cast<size_t>(tr->rt) * D);
    for (int b = 0; b < tr->nr; ++b) elems.insert(elems.end(), blk, blk + kBlockEntries);
    elems.insert(elems.end(), {D, D * D, D, static_cast<size_t>(tr->Cr) * D,
                               static_cast<size_t>(tr->Cr)});
    if (elems.size() != n_ent) {
      delete tr;
      return FD_ERR_CONFIG;
    }
    size_t off = 0;
    for (size_t e : elems) {
      tr->goff.push_back(off);
      off += e;
    }
  }
  bool ok = true;
  const int D = tr->D, Dm = tr->Dm, QO = tr->QO, NQ = tr->NQ, G = tr->G, MB = tr->MB,
            MR = tr->MR;
  const int Mmax = MB > MR ? MB : MR;
  const int Pmax = tr->rt > 1 ? tr->rt * tr->Lp : tr->Lp;
  const int Kmax = std::min(tr->T, tr->Wn) * Pmax;  // keys of one query chunk's window
  // heads per attention product: all of a KV group's, unless S (fp32 [heads Pmax][Kmax]) would
  // pass 512 M elements; then the largest divisor of the group size that stays within it
  {
    const int hpg = tr->N / tr->G;
    tr->hs = 1;
    for (int d = hpg; d >= 1; --d)
      if (hpg % d == 0 && static_cast<size_t>(d) * Pmax * Kmax <= (static_cast<size_t>(1) << 29)) {
        tr->hs = d;
        break;
      }
  }
  const size_t RK = static_cast<size_t>(tr->hs) * Pmax * Kmax;  // one product's scores
  tr->err = dalloc<int>(tr, 4, ok);
  tr->zero_bias = dalloc<float>(tr, std::max({Kmax, Dm, QO, NQ, tr->rt * D, tr->Cr, D}), ok);
  // RoPE tables, fp64 on the host (frames 0 .. T r_t - 1; rows; columns)
  {
    const int F = tr->T * tr->rt;
    const double base = cfg->rope_base;
    std::vector<float2> ht(static_cast<size_t>(F) * fd::train::kBandT),
        hy(static_cast<size_t>(tr->gh) * fd::train::kBandS),
        hx(static_cast<size_t>(tr->gw) * fd::train::kBandS);
    for (int f = 0; f < F; ++f)
      for (int i = 0; i < fd::train::kBandT; ++i) {
        const double a = f * rope_inv_freq(i, base);
        ht[f * fd::train::kBandT + i] = make_float2(static_cast<float>(std::cos(a)),
                                                    static_cast<float>(std::sin(a)));
      }
    for (int y = 0; y < tr->gh; ++y)
      for (int i = 0; i < fd::train::kBandS; ++i) {
        const double a = y * rope_inv_freq(fd::train::kBandT + i, base);
        hy[y * fd::train::kBandS + i] = make_float2(static_cast<float>(std::cos(a)),
                                                    static_cast<float>(std::sin(a)));
      }
    for (int x = 0; x < tr->gw; ++x)
      for (int i = 0; i < fd::train::kBandS; ++i) {
        const double a = x * rope_inv_freq(fd::train::kBandT + fd::train::kBandS + i, base);
        hx[x * fd::train::kBandS + i] = make_float2(static_cast<float>(std::cos(a)),
                                                    static_cast<float>(std::sin(a)));
      }
    tr->rope_t = dalloc<float2>(tr, ht.size(), ok);
    tr->rope_y = dalloc<float2>(tr, hy.size(), ok);
    tr->rope_x = dalloc<float2>(tr, hx.size(), ok);
    if (ok)
      ok = cudaMemcpy(tr->rope_t, ht.data(), ht.size() * sizeof(float2), cudaMemcpyHostToDevice) ==
               cudaSuccess &&
           cudaMemcpy(tr->rope_y, hy.data(), hy.size() * sizeof(float2), cudaMemcpyHostToDevice) ==
               cudaSuccess &&
           cudaMemcpy(tr->rope_x, hx.data(), hx.size() * sizeof(float2), cudaMemcpyHostToDevice) ==
               cudaSuccess;
  }
  auto alloc_stack = [&](fd_trainer_s::Stack& st, int M, int Pc, int nblocks) {
    st.M = M;
    st.Pc = Pc;
    for (int b = 0; b <= nblocks; ++b) st.h.push_back(dalloc<float>(tr, static_cast<size_t>(M) * D, ok));
    for (int b = 0; b < nblocks; ++b) {
      st.u.push_back(dalloc<bf16>(tr, static_cast<size_t>(M) * D, ok));
      st.qkv.push_back(dalloc<float>(tr, static_cast<size_t>(M) * QO, ok));
      st.q2.push_back(dalloc<bf16>(tr, static_cast<size_t>(M) * NQ, ok));
      st.k2.push_back(dalloc<bf16>(tr, static_cast<size_t>(G) * M * 64, ok));
      st.v1.push_back(dalloc<bf16>(tr, static_cast<size_t>(G) * M * 64, ok));
      st.lse.push_back(dalloc<float>(tr, static_cast<size_t>(M) * tr->N, ok));
      st.o.push_back(dalloc<bf16>(tr, static_cast<size_t>(M) * NQ, ok));
      st.hm.push_back(dalloc<float>(tr, static_cast<size_t>(M) * D, ok));
      st.u2.push_back(dalloc<bf16>(tr, static_cast<size_t>(M) * D, ok));
      st.z.push_back(dalloc<float>(tr, static_cast<size_t>(M) * tr->Dz, ok));
      st.a.push_back(dalloc<bf16>(tr, static_cast<size_t>(M) * Dm, ok));
    }
  };
  alloc_stack(tr->sB, MB, tr->Lp, tr->nb);
  alloc_stack(tr->sR, MR, tr->rt * tr->Lp, tr->nr);
  // the forward's band attention: per stack, the query rows, unpadded K / V^T (allocated
  // zeroed: keys past the clip read zeros), the kernel's per-chunk stream table and its
  // workspace (counters zero); else the materialised forward with its head-major O scratch
  int sms = 0, dev = 0;
  if (ok) ok = cudaGetDevice(&dev) == cudaSuccess &&
               cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess;
  auto setup_band = [&](fd_trainer_s::Stack& st, int Lu) {
    auto& bd = st.band;
    const int T = tr->T, M = st.M;
    bd.Lu = Lu;
    bd.pitch = (T * Lu + 127) / 128 * 128;
    bd.on = ok && (Lu % 8 == 0 || T == 1);
    if (bd.on) {
      bd.qr = dalloc<bf16>(tr, static_cast<size_t>(M) * NQ, ok);
      bd.k = dalloc<bf16>(tr, static_cast<size_t>(G) * bd.pitch * 64, ok);
      bd.vt = dalloc<__half>(tr, static_cast<size_t>(G) * 64 * bd.pitch, ok);
      bd.steps = dalloc<int>(tr, T, ok);
      bd.streams = dalloc<fd::AttnStream>(tr, T, ok);
      const int keys = std::min(T, tr->Wn) * Lu;
      bd.pairs = fd::attention_units(st.Pc, tr->N, G);
      const long long units = static_cast<long long>(bd.pairs) * ((keys + 127) / 128);
      bd.parts = static_cast<int>(std::max(1LL, std::min<long long>(std::max(1, sms / T), units)));
      bd.ws_stride = (fd::attention_workspace_floats(bd.parts, bd.pairs) + 63) / 64 * 64;
      bd.ws = dalloc<float>(tr, bd.ws_stride * T, ok);
    }
    if (bd.on && ok) {
      std::vector<fd::AttnStream> host(T);
      std::vector<int> steps(T);
      for (int i = 0; i < T; ++i) steps[i] = i;
      bd.on = fd::band_attention_maps(host.data(), T, tr->Wn, Lu, G, bd.pitch, bd.k, bd.vt,
                                      bd.steps, tr->err) &&
              fd::attention_q_maps(&bd.tmQ, &bd.tmQ8, bd.qr, M, tr->N);
      if (bd.on)
        ok = cudaMemcpy(bd.streams, host.data(), T * sizeof(fd::AttnStream),
                        cudaMemcpyHostToDevice) == cudaSuccess &&
             cudaMemcpy(bd.steps, steps.data(), T * sizeof(int), cudaMemcpyHostToDevice) ==
                 cudaSuccess;
    }
    if (!bd.on) st.o32 = dalloc<float>(tr, static_cast<size_t>(M) * NQ, ok);
  };
  setup_band(tr->sB, tr->L);
  setup_band(tr->sR, tr->rt * tr->L);
  const size_t wide = static_cast<size_t>(Mmax) *
                      std::max({D, tr->Dz, QO, NQ, tr->rt * D, tr->Cr});
  tr->x0 = dalloc<bf16>(tr, static_cast<size_t>(MB) * tr->cin, ok);
  tr->y16 = dalloc<bf16>(tr, static_cast<size_t>(MB) * D, ok);
  tr->yh16 = dalloc<bf16>(tr, static_cast<size_t>(MR) * D, ok);
  tr->a1 = dalloc<bf16>(tr, static_cast<size_t>(MR) * D, ok);
  tr->vT = dalloc<bf16>(tr, static_cast<size_t>(G) * 64 * Mmax, ok);
  tr->kT = dalloc<bf16>(tr, static_cast<size_t>(G) * 64 * Mmax, ok);
  tr->do16 = dalloc<bf16>(tr, static_cast<size_t>(Mmax) * NQ, ok);
  tr->dS = dalloc<bf16>(tr, RK, ok);
  // S and P of the materialised forward (a stack whose band attention is off)
  const bool materialised = !tr->sB.band.on || !tr->sR.band.on;
  if (materialised) tr->P16 = dalloc<bf16>(tr, RK, ok);
  tr->dST = dalloc<bf16>(tr, RK, ok);
  tr->PT = dalloc<bf16>(tr, RK, ok);
  tr->QT = dalloc<bf16>(tr, static_cast<size_t>(64) * tr->hs * Pmax, ok);
  tr->dOT = dalloc<bf16>(tr, static_cast<size_t>(64) * tr->hs * Pmax, ok);
  tr->dy16 = dalloc<bf16>(tr, wide, ok);
  tr->dyT = dalloc<bf16>(tr, wide, ok);
  tr->xT = dalloc<bf16>(tr, wide, ok);
  tr->dqkv16 = dalloc<bf16>(tr, wide, ok);
  tr->e = dalloc<float>(tr, static_cast<size_t>(MB) * tr->rt * D, ok);
  tr->z1 = dalloc<float>(tr, static_cast<size_t>(MR) * D, ok);
  tr->F = dalloc<float>(tr, static_cast<size_t>(MR) * tr->Cr, ok);
  tr->dF = dalloc<float>(tr, static_cast<size_t>(MR) * tr->Cr, ok);
  tr->loss_blocks = static_cast<int>((static_cast<long long>(MR) * tr->Cr + 255) / 256);
  tr->loss_part = dalloc<float>(tr, tr->loss_blocks, ok);
  if (materialised) tr->S = dalloc<float>(tr, RK, ok);
  tr->delta = dalloc<float>(tr, static_cast<size_t>(Mmax) * tr->N, ok);
  {
    const size_t R = fd::train::kColsumRows;
    const size_t widest = std::max({D, tr->Dz, QO, NQ, tr->rt * D, tr->Cr});
    tr->colsum_elems = std::max((static_cast<size_t>(Mmax) * tr->N + R - 1) / R * 64,
                                (static_cast<size_t>(Mmax) + R - 1) / R * widest);
    tr->colsum_part = dalloc<float>(tr, tr->colsum_elems, ok);
  }
  tr->dq2 = dalloc<float>(tr, static_cast<size_t>(Mmax) * NQ, ok);
  tr->dk2 = dalloc<float>(tr, static_cast<size_t>(G) * Mmax * 64, ok);
  tr->dv1 = dalloc<float>(tr, static_cast<size_t>(G) * Mmax * 64, ok);
  tr->dqkv = dalloc<float>(tr, static_cast<size_t>(Mmax) * QO, ok);
  tr->tq = dalloc<float>(tr, static_cast<size_t>(Mmax) * tr->N * 64, ok);
  tr->tk = dalloc<float>(tr, static_cast<size_t>(Mmax) * G * 64, ok);
  tr->tv = dalloc<float>(tr, static_cast<size_t>(Mmax) * G * 64, ok);
  tr->gA = dalloc<float>(tr, wide, ok);
  tr->gB = dalloc<float>(tr, wide, ok);
  tr->gC = dalloc<float>(tr, wide, ok);
  tr->tbuf = dalloc<float>(tr, static_cast<size_t>(Mmax) * D, ok);
  tr->gtmp = dalloc<float>(tr, static_cast<size_t>(D) * std::max({D, tr->Dz, QO, tr->Cr, tr->cin}),
                           ok);
  if (tr->gated) {
    tr->dz32 = dalloc<float>(tr, static_cast<size_t>(Mmax) * tr->Dz, ok);
    tr->dwz = dalloc<float>(tr, static_cast<size_t>(tr->Dz) * (D + 1), ok);
  }
  // transposed weights [in][out] for the input gradients dX = dY W
  auto wT = [&](size_t entry, int n_out, int n_in) -> bf16* {
    bf16* t = dalloc<bf16>(tr, static_cast<size_t>(n_out) * n_in, ok);
    if (ok) {
      dim3 grid((n_in + 31) / 32, (n_out + 31) / 32);
      fd::train::transpose_kernel<bf16><<<grid, dim3(32, 8)>>>(
          static_cast<const bf16*>(tr->wt[entry]), n_out, n_in, n_in, t, n_out);
      ok = cudaGetLastError() == cudaSuccess;
    }
    return t;
  };
  auto stackT = [&](std::vector<fd_trainer_s::LinT>& v, size_t e0, int nblocks) {
    for (int b = 0; b < nblocks; ++b) {
      const size_t e = e0 + static_cast<size_t>(b) * kBlockEntries;
      v.push_back({wT(e + kQW, QO, D), wT(e + kOW, D, NQ), wT(e + kM1W, tr->Dz, D),
                   wT(e + kM2W, D, Dm)});
    }
  };
  const size_t eB = 2, eF = eB + static_cast<size_t>(tr->nb) * kBlockEntries;
  const size_t eR = eF + 3, eH = eR + static_cast<size_t>(tr->nr) * kBlockEntries;
  stackT(tr->tB, eB, tr->nb);
  tr->t_tup = wT(eF + 1, tr->rt * D, D);
  stackT(tr->tR, eR, tr->nr);
  tr->t_head1 = wT(eH + 1, D, D);
  tr->t_head2 = wT(eH + 3, tr->Cr, D);
  if (ok) ok = cudaDeviceSynchronize() == cudaSuccess;
  if (!ok) {
    for (void* ptr : tr->allocs) cudaFree(ptr);
    delete tr;
    return FD_ERR_OOM;
  }
  fd::weights_add_user(w, 1);
  *out = tr;
  return FD_OK;
}

fd_status fd_train_step(fd_trainer tr, const float* latents, const float* targets, float* loss,
                        float* grads, void* stream) {
  if (tr == nullptr || latents == nullptr || targets == nullptr || loss == nullptr ||
      grads == nullptr)
    return FD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(latents) | reinterpret_cast<uintptr_t>(targets) |
       reinterpret_cast<uintptr_t>(grads)) & 15u)
    return FD_ERR_INVALID_ARG;
  Run r{tr, static_cast<cudaStream_t>(stream)};
  const int D = tr->D, MB = tr->MB, MR = tr->MR, rt = tr->rt;
  const size_t eB = 2, eF = eB + static_cast<size_t>(tr->nb) * kBlockEntries;
  const size_t eR = eF + 3, eH = eR + static_cast<size_t>(tr->nr) * kBlockEntries;
  if (r.begin(FD_TK_POINTWISE)) {
    r.check(cudaMemsetAsync(tr->err, 0, sizeof(int), r.s));
    r.end();
  }
  // ---- forward
  // patch-embedding (Eq. projection) of every chunk: PixelUnshuffle rows, then the linear
  const size_t chw = static_cast<size_t>(tr->C) * tr->H * tr->W;
  for (int c = 0; c < tr->T && r.begin(FD_TK_POINTWISE); ++c) {
    r.check(fd::launch_unshuffle(latents + c * chw, tr->C, tr->H, tr->W, tr->p,
                                 tr->x0 + static_cast<size_t>(c) * tr->Lp * tr->cin, r.s));
    r.end();
  }
  r.gemm(FD_TK_LINEAR, fd::EPI_F32, MB, D, tr->cin, tr->x0, tr->cin, r.wb(0), tr->cin, r.wf(1), tr->sB.h[0], D);
  for (int b = 0; b < tr->nb; ++b)
    block_fwd(r, tr->sB, b, eB + static_cast<size_t>(b) * kBlockEntries);
  // final norm and temporal upsampling (Eq. temporal_upsample): channel block tau -> frame tau
  const float* hBo = tr->sB.h[tr->nb];
  r.rmsnorm(hBo, r.wf(eF), MB, tr->y16);
  r.gemm(FD_TK_LINEAR, fd::EPI_F32, MB, rt * D, D, tr->y16, D, r.wb(eF + 1), D, r.wf(eF + 2), tr->e, rt * D);
  if (r.begin(FD_TK_POINTWISE)) {
    const long long n = static_cast<long long>(MB) * rt * D;
    fd::train::tup_permute_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(
        tr->e, tr->T, rt, tr->Lp, D, 0, tr->sR.h[0], nullptr);
    r.check(cudaGetLastError());
    r.end();
  }
  for (int b = 0; b < tr->nr; ++b)
    block_fwd(r, tr->sR, b, eR + static_cast<size_t>(b) * kBlockEntries);
  // head (Sec. 3.4 Step 3): RMSNorm, Linear + GELU, Linear to C r_s^2 per refined token
  const float* hRo = tr->sR.h[tr->nr];
  r.rmsnorm(hRo, r.wf(eH), MR, tr->yh16);
  r.gemm(FD_TK_LINEAR, fd::EPI_F32, MR, D, D, tr->yh16, D, r.wb(eH + 1), D, r.wf(eH + 2), tr->z1, D);
  if (r.begin(FD_TK_POINTWISE)) {
    const long long n = static_cast<long long>(MR) * D;
    fd::train::gelu_fwd_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(tr->z1, n, tr->a1);
    r.check(cudaGetLastError());
    r.end();
  }
  r.gemm(FD_TK_LINEAR, fd::EPI_F32, MR, tr->Cr, D, tr->a1, D, r.wb(eH + 3), D, r.wf(eH + 4), tr->F, tr->Cr);
  // ---- loss (L1 over every pixel of the clip) and its gradient through the pixel shuffle
  const int first = tr->f1 ? 1 : rt;  // frames chunk 0 emits (reading R16)
  const double total = (static_cast<double>(tr->T - 1) * rt + first) * tr->Cout * tr->gh *
                       tr->rs * tr->gw * tr->rs;
  const float inv_total = static_cast<float>(1.0 / total);
  if (r.begin(FD_TK_POINTWISE)) {
    fd::train::l1_head_kernel<<<tr->loss_blocks, 256, 0, r.s>>>(
        tr->F, targets, tr->T, rt, first, tr->Lp, tr->L, tr->gh, tr->gw, tr->Cout, tr->rs,
        inv_total, tr->dF, tr->loss_part);
    r.check(cudaGetLastError());
    r.end();
  }
  if (r.begin(FD_TK_POINTWISE)) {
    fd::train::finish_loss_kernel<<<1, fd::train::kLossThreads, 0, r.s>>>(tr->loss_part,
                                                                         tr->loss_blocks, inv_total,
                                                     loss);
    r.check(cudaGetLastError());
    r.end();
  }
  // ---- backward
  float* g = grads;
  // head layer 2
  r.bf(tr->dF, static_cast<long long>(MR) * tr->Cr, tr->dy16);
  r.gemm(FD_TK_DGRAD, fd::EPI_F32, MR, D, tr->Cr, tr->dy16, tr->Cr, tr->t_head2, tr->Cr, nullptr, tr->gC, D);
  r.wgrad(tr->dy16, tr->Cr, tr->a1, D, MR, r.grad(g, eH + 3));
  r.colsum(tr->dF, MR, tr->Cr, tr->Cr, r.grad(g, eH + 4));
  // head layer 1 (GELU')
  if (r.begin(FD_TK_POINTWISE)) {
    const long long n = static_cast<long long>(MR) * D;
    fd::train::gelu_bwd_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(tr->z1, tr->gC, n, tr->gC,
                                                                      tr->dqkv16);
    r.check(cudaGetLastError());
    r.end();
  }
  r.gemm(FD_TK_DGRAD, fd::EPI_F32, MR, D, D, tr->dqkv16, D, tr->t_head1, D, nullptr, tr->gA, D);
  r.wgrad(tr->dqkv16, D, tr->yh16, D, MR, r.grad(g, eH + 1));
  r.colsum(tr->gC, MR, D, D, r.grad(g, eH + 2));
  // the head's RMSNorm
  r.rmsnorm_bwd(hRo, r.wf(eH), tr->gA, nullptr, MR, tr->gB, r.grad(g, eH));
  for (int b = tr->nr - 1; b >= 0; --b)
    block_bwd(r, tr->sR, b, eR + static_cast<size_t>(b) * kBlockEntries, tr->tR[b], g);
  // temporal upsampling: refined frame tau back to channel block tau
  if (r.begin(FD_TK_POINTWISE)) {
    const long long n = static_cast<long long>(MB) * rt * D;
    fd::train::tup_permute_kernel<<<blocks_for(n, 256), 256, 0, r.s>>>(
        tr->gB, tr->T, rt, tr->Lp, D, 1, tr->gC, tr->dqkv16);
    r.check(cudaGetLastError());
    r.end();
  }
  r.gemm(FD_TK_DGRAD, fd::EPI_F32, MB, D, rt * D, tr->dqkv16, rt * D, tr->t_tup, rt * D, nullptr, tr->gA, D);
  r.wgrad(tr->dqkv16, rt * D, tr->y16, D, MB, r.grad(g, eF + 1));
  r.colsum(tr->gC, MB, rt * D, rt * D, r.grad(g, eF + 2));
  r.rmsnorm_bwd(hBo, r.wf(eF), tr->gA, nullptr, MB, tr->gB, r.grad(g, eF));
  for (int b = tr->nb - 1; b >= 0; --b)
    block_bwd(r, tr->sB, b, eB + static_cast<size_t>(b) * kBlockEntries, tr->tB[b], g);
  // patch-embedding: weight and bias gradients only
  r.bf(tr->gB, static_cast<long long>(MB) * D, tr->dy16);
  r.wgrad(tr->dy16, D, tr->x0, tr->cin, MB, r.grad(g, 0));
  r.colsum(tr->gB, MB, D, D, r.grad(g, 1));
  return r.ok ? FD_OK : FD_ERR_CUDA;
}

// ---- single kernels of the step, for per-kernel checks (include/flashdec_ops.h)
fd_status fd_op_scores_bwd(int M, int N, const void* Q, const void* dO, const void* K,
                           const void* V, const float* lse, const float* delta, int Pc, int Lp,
                           int L, void* dS, void* dST, void* PT, int* err_dev, void* stream) {
  if (!Q || !dO || !K || !V || !lse || !delta || !dS || !dST || !PT || !err_dev || M < 1 ||
      N < 32 || N % 32 || Lp < 1 || Pc < Lp || Pc % Lp || L < 1 || L > Lp)
    return FD_ERR_INVALID_ARG;
  const void* const ptrs[7] = {Q, dO, K, V, dS, dST, PT};
  for (const void* ptr : ptrs)
    if (reinterpret_cast<uintptr_t>(ptr) & 15u) return FD_ERR_INVALID_ARG;
  const fd::DsEpi ds{lse, delta, 0.125f, Pc, Lp, L, static_cast<bf16*>(dS),
                     static_cast<bf16*>(dST), static_cast<bf16*>(PT)};
  const cudaError_t e = fd::scores_bwd(M, N, static_cast<const bf16*>(Q),
                                       static_cast<const bf16*>(dO), 64,
                                       static_cast<const bf16*>(K), static_cast<const bf16*>(V),
                                       64, ds, err_dev, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FD_OK : FD_ERR_CUDA;
}

fd_status fd_op_rmsnorm_bwd(const float* x, const float* g, const float* dy, int M, int D,
                            float eps, float* dx, float* dg, float* work, void* stream) {
  if (!x || !g || !dy || !dx || !dg || !work || M < 1 || D < 1 || D > 65536)
    return FD_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  fd::train::rmsnorm_bwd_kernel<<<(M + 7) / 8, 256, 0, s>>>(x, g, dy, nullptr, M, D, eps, dx,
                                                            work);
  if (cudaGetLastError() != cudaSuccess) return FD_ERR_CUDA;
  fd::train::colsum_kernel<<<(D + 127) / 128, 128, 0, s>>>(work, M, D, D, dg);
  return cudaGetLastError() == cudaSuccess ? FD_OK : FD_ERR_CUDA;
}

fd_status fd_op_gelu_bwd(const float* z, const float* da, int64_t n, float* dz, void* dz_bf16,
                         void* stream) {
  if (!z || !da || !dz || !dz_bf16 || n < 1) return FD_ERR_INVALID_ARG;
  fd::train::gelu_bwd_kernel<<<blocks_for(n, 256), 256, 0, static_cast<cudaStream_t>(stream)>>>(
      z, da, n, dz, static_cast<bf16*>(dz_bf16));
  return cudaGetLastError() == cudaSuccess ? FD_OK : FD_ERR_CUDA;
}

fd_status fd_op_l1_pixel_bwd(const float* F, const float* target, int frames, int grid_h,
                             int grid_w, int channels, int rs, float* dF, float* loss,
                             float* work, void* stream) {
  if (!F || !target || !dF || !loss || !work || frames < 1 || grid_h < 1 || grid_w < 1 ||
      channels < 1 || rs < 1)
    return FD_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int L = grid_h * grid_w;
  const long long n = static_cast<long long>(frames) * L * channels * rs * rs;
  const int blocks = static_cast<int>((n + 255) / 256);
  const float inv_total = static_cast<float>(1.0 / static_cast<double>(n));
  // one chunk of `frames` refined frames, rows unpadded (Lp = L)
  fd::train::l1_head_kernel<<<blocks, 256, 0, s>>>(F, target, 1, frames, frames, L, L, grid_h,
                                                   grid_w, channels, rs, inv_total, dF, work);
  if (cudaGetLastError() != cudaSuccess) return FD_ERR_CUDA;
  fd::train::finish_loss_kernel<<<1, fd::train::kLossThreads, 0, s>>>(work, blocks, inv_total,
                                                                       loss);
  return cudaGetLastError() == cudaSuccess ? FD_OK : FD_ERR_CUDA;
}

fd_status fd_train_status(fd_trainer tr, void* stream) {
  if (tr == nullptr) return FD_ERR_INVALID_ARG;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return FD_ERR_CUDA;
  int e = 0;
  if (cudaMemcpy(&e, tr->err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return FD_ERR_CUDA;
  return e ? FD_ERR_DEVICE_TIMEOUT : FD_OK;
}

fd_status fd_train_profile_enable(fd_trainer tr, int enable) {
  if (tr == nullptr) return FD_ERR_INVALID_ARG;
  tr->prof = enable != 0;
  return FD_OK;
}

fd_status fd_train_profile_collect(fd_trainer tr, int64_t* launches, double* ms) {
  if (tr == nullptr || launches == nullptr || ms == nullptr) return FD_ERR_INVALID_ARG;
  if (cudaDeviceSynchronize() != cudaSuccess) return FD_ERR_CUDA;
  fd_status st = FD_OK;
  for (const fd_trainer_s::Rec& e : tr->rec) {
    float t = 0.f;
    if (cudaEventElapsedTime(&t, e.a, e.b) != cudaSuccess) st = FD_ERR_CUDA;
    if (e.kind >= 0 && e.kind < FD_TK_COUNT) {
      launches[e.kind] += 1;
      ms[e.kind] += t;
    }
    tr->ev_free.push_back(e.a);
    tr->ev_free.push_back(e.b);
  }
  tr->rec.clear();
  return st;
}

fd_status fd_train_destroy(fd_trainer tr) {
  if (tr == nullptr) return FD_ERR_INVALID_ARG;
  cudaDeviceSynchronize();
  for (cudaEvent_t e : tr->ev_all) cudaEventDestroy(e);
  for (void* ptr : tr->allocs) cudaFree(ptr);
  fd::weights_add_user(tr->w, -1);
  delete tr;
  return FD_OK;
}

}  // extern "C"
