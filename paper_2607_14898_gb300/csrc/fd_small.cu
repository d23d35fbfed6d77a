// Bandwidth-bound kernels of the decode path.
//   unshuffle    latent [C'][H'][W'] fp32 -> tokens [L][C' p^2] bf16 (PixelUnshuffle, Sec. 4.3;
//                raster token order of Eq. projection)
//   rmsnorm      h fp32 [M][D] -> bf16(h / sqrt(mean(h^2) + eps) * g)  (pre-norm, Sec. 3.2),
//                or e4m3 of that times a scale (input of an FP8 MLP)
//   pixel_head   F fp32 [frames*L][C r_s^2] -> PixelShuffle(r_s) + clamp to [-1, 1], fp32 or
//                uint8 (Sec. 3.4 "Step 3"); one thread per 4 consecutive output pixels
//   kv_append    fp32 K, V of one chunk -> ring slot (K rows bf16, V transposed fp16) (Sec. 3.3)
//   advance      chunk counter t += 1 (device-resident, so a captured graph can be replayed)
//   wait_check   failure-path check: a wait on an mbarrier that nothing arrives at, through
//                the decode kernels' bounded wait, gives up after a short limit and returns
#include "fd_internal.h"
#include "fd_ptx.cuh"

namespace fd {

__global__ void unshuffle_kernel(const float* __restrict__ z, int C, int H, int W, int p,
                                 __nv_bfloat16* __restrict__ x0) {
  grid_dep_wait();
  grid_dep_launch();
  const int gw = W / p;
  const int cin = C * p * p;
  const int total = (H / p) * gw * cin;
  for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += gridDim.x * blockDim.x) {
    const int l = idx / cin, ch = idx - l * cin;
    const int c = ch / (p * p), ij = ch - c * p * p;
    const int i = ij / p, j = ij - i * p;
    const int h = l / gw, w = l - h * gw;
    x0[idx] = __float2bfloat16_rn(z[(static_cast<size_t>(c) * H + h * p + i) * W + w * p + j]);
  }
}

// one warp per row, the row held in registers (D / 128 float4 per lane for D / 128 in
// {2, 4, 8, 12, 16}, one pass over h; any other multiple of 128 takes two passes); output bf16,
// or e4m3 of (y * oscale) when F8
template <int CH, bool F8>
__device__ __forceinline__ void rmsnorm_row(const float4* hr, const float4* g4, int lane,
                                            float inv_d, float eps, void* out_row,
                                            float oscale) {
  float4 v[CH];
  float ss = 0.f;
#pragma unroll
  for (int c = 0; c < CH; ++c) {
    v[c] = hr[lane + 32 * c];
    ss = fmaf(v[c].x, v[c].x, fmaf(v[c].y, v[c].y, fmaf(v[c].z, v[c].z, fmaf(v[c].w, v[c].w, ss))));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float r = rsqrtf(ss * inv_d + eps);
#pragma unroll
  for (int c = 0; c < CH; ++c) {
    const float4 gg = g4[lane + 32 * c];
    const float y0 = v[c].x * r * gg.x, y1 = v[c].y * r * gg.y;
    const float y2 = v[c].z * r * gg.z, y3 = v[c].w * r * gg.w;
    if (F8) {
      reinterpret_cast<uint32_t*>(out_row)[lane + 32 * c] =
          pack_e4m3x4(y0 * oscale, y1 * oscale, y2 * oscale, y3 * oscale);
    } else {
      reinterpret_cast<uint2*>(out_row)[lane + 32 * c] =
          make_uint2(pack_bf16x2(y0, y1), pack_bf16x2(y2, y3));
    }
  }
}

template <bool F8>
__global__ void rmsnorm_kernel(const float* __restrict__ h, const float* __restrict__ g, int M,
                               int D, float eps, void* __restrict__ u, float oscale) {
  grid_dep_wait();
  grid_dep_launch();
  const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= M) return;
  const float4* hr = reinterpret_cast<const float4*>(h + static_cast<size_t>(row) * D);
  const float4* g4 = reinterpret_cast<const float4*>(g);
  void* ur = static_cast<uint8_t*>(u) + static_cast<size_t>(row) * D * (F8 ? 1 : 2);
  const float inv_d = 1.0f / static_cast<float>(D);
  switch (D / 128) {  // chunks of 128 elements per lane-row
    case 2: rmsnorm_row<2, F8>(hr, g4, lane, inv_d, eps, ur, oscale); break;
    case 4: rmsnorm_row<4, F8>(hr, g4, lane, inv_d, eps, ur, oscale); break;
    case 8: rmsnorm_row<8, F8>(hr, g4, lane, inv_d, eps, ur, oscale); break;
    case 12: rmsnorm_row<12, F8>(hr, g4, lane, inv_d, eps, ur, oscale); break;
    case 16: rmsnorm_row<16, F8>(hr, g4, lane, inv_d, eps, ur, oscale); break;
    default: {  // any other multiple of 128: two passes
      float ss = 0.f;
      for (int c = lane; c < D / 4; c += 32) {
        const float4 v = hr[c];
        ss = fmaf(v.x, v.x, fmaf(v.y, v.y, fmaf(v.z, v.z, fmaf(v.w, v.w, ss))));
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
      const float r = rsqrtf(ss * inv_d + eps);
      for (int c = lane; c < D / 4; c += 32) {
        const float4 v = hr[c];
        const float4 gg = g4[c];
        const float y0 = v.x * r * gg.x, y1 = v.y * r * gg.y;
        const float y2 = v.z * r * gg.z, y3 = v.w * r * gg.w;
        if (F8) {
          reinterpret_cast<uint32_t*>(ur)[c] =
              pack_e4m3x4(y0 * oscale, y1 * oscale, y2 * oscale, y3 * oscale);
        } else {
          reinterpret_cast<uint2*>(ur)[c] = make_uint2(pack_bf16x2(y0, y1), pack_bf16x2(y2, y3));
        }
      }
    }
  }
}


// pix[c][tau][y][x] = clamp(F[tau*L + (y/rs)*gw + x/rs][c*rs*rs + (y%rs)*rs + x%rs]); rs % 4 == 0
// frame tau's tokens are rows tau * frame_rows .. + gh gw - 1 of F (frame_rows >= gh gw)
__global__ void pixel_head_kernel(const float* __restrict__ F, int frames, int frame_rows, int gh,
                                  int gw, int C, int rs, int out_u8, void* __restrict__ pix) {
  grid_dep_wait();
  grid_dep_launch();
  const int Wo = gw * rs, Ho = gh * rs;
  const int ld = C * rs * rs;
  const int q_per_row = Wo / 4;
  const long long total = static_cast<long long>(C) * frames * Ho * q_per_row;
  for (long long idx = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
       idx < total; idx += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int xq = static_cast<int>(idx % q_per_row);
    long long r = idx / q_per_row;
    const int y = static_cast<int>(r % Ho);
    r /= Ho;
    const int tau = static_cast<int>(r % frames);
    const int c = static_cast<int>(r / frames);
    const int x = 4 * xq;
    const int tok = tau * frame_rows + (y / rs) * gw + x / rs;
    const int ch = c * rs * rs + (y % rs) * rs + (x % rs);
    const float4 v = *reinterpret_cast<const float4*>(F + static_cast<size_t>(tok) * ld + ch);
    const size_t o = ((static_cast<size_t>(c) * frames + tau) * Ho + y) * Wo + x;
    if (out_u8) {
      const uint32_t packed = quant_u8(v.x) | (quant_u8(v.y) << 8) | (quant_u8(v.z) << 16) |
                              (quant_u8(v.w) << 24);
      *reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(pix) + o) = packed;
    } else {
      *reinterpret_cast<float4*>(static_cast<float*>(pix) + o) =
          make_float4(fminf(fmaxf(v.x, -1.f), 1.f), fminf(fmaxf(v.y, -1.f), 1.f),
                      fminf(fmaxf(v.z, -1.f), 1.f), fminf(fmaxf(v.w, -1.f), 1.f));
    }
  }
}

// K, V fp32 [groups][rows][64] -> k_ring[g][slot*rows + r][d] (bf16) and
// vt_ring[g][d][slot*rows + r] (fp16), both rounded to nearest even. Block: 32 x 8 threads over a 32-row x 64-dim tile; V goes
// through shared memory so both the read and the transposed write are coalesced.
__global__ void kv_append_kernel(const float* __restrict__ k, const float* __restrict__ v,
                                 int rows, int slot, int pitch, __nv_bfloat16* __restrict__ k_ring,
                                 __half* __restrict__ vt_ring) {
  __shared__ float tile[64][33];
  grid_dep_wait();
  grid_dep_launch();
  const int g = blockIdx.y;
  const int r0 = blockIdx.x * 32;
  const size_t src = static_cast<size_t>(g) * rows * kHeadDim;
  const size_t dst_row0 = static_cast<size_t>(g) * pitch + static_cast<size_t>(slot) * rows;
  for (int rr = threadIdx.y; rr < 32; rr += blockDim.y) {
    const int r = r0 + rr;
    if (r >= rows) break;
    for (int d = threadIdx.x; d < kHeadDim; d += 32) {
      k_ring[(dst_row0 + r) * kHeadDim + d] = __float2bfloat16_rn(k[src + r * kHeadDim + d]);
      tile[d][rr] = v[src + static_cast<size_t>(r) * kHeadDim + d];
    }
  }
  __syncthreads();
  for (int d = threadIdx.y; d < kHeadDim; d += blockDim.y) {
    const int r = r0 + threadIdx.x;
    if (r < rows)
      vt_ring[(static_cast<size_t>(g) * kHeadDim + d) * pitch + slot * static_cast<size_t>(rows) +
              r] = __float2half_rn(tile[d][threadIdx.x]);
  }
}

__global__ void advance_kernel(int* step) {
  grid_dep_wait();
  grid_dep_launch();
  *step += 1;
}

struct RopeSets {
  int frames[kMaxRopeSets];
  double inv_freq[kRopePairs];
};

// one thread per (set, frame, pair): angles reduced and evaluated in fp64, stored as fp32
__global__ void rope_table_kernel(const int* step_dev, int t_host, int nsets, int band_t,
                                  RopeSets sets, float2* table) {
  grid_dep_wait();
  grid_dep_launch();
  const int t = step_dev ? *step_dev : t_host;
  int off = 0;
  for (int k = 0; k < nsets; ++k) {
    const int n = sets.frames[k] * band_t;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
      const int tau = i / band_t, pair = i - tau * band_t;
      const double f = static_cast<double>(t) * sets.frames[k] + tau;
      double sn, cs;
      sincos(f * sets.inv_freq[pair], &sn, &cs);
      table[off + i] = make_float2(static_cast<float>(cs), static_cast<float>(sn));
    }
    off += n;
  }
}

static int grid_for(long long work, int threads) {
  long long b = (work + threads - 1) / threads;
  if (b > 152LL * 16) b = 152LL * 16;
  return static_cast<int>(b < 1 ? 1 : b);
}

cudaError_t launch_unshuffle(const float* z, int C, int H, int W, int p, __nv_bfloat16* x0,
                             cudaStream_t s) {
  const long long total = static_cast<long long>(H / p) * (W / p) * C * p * p;
  return launch_pdl(unshuffle_kernel, dim3(grid_for(total, 256)), dim3(256), 0, s, z, C, H, W, p,
                    x0);
}

cudaError_t launch_rmsnorm(const float* h, const float* g, int M, int D, float eps,
                           __nv_bfloat16* u, cudaStream_t s) {
  return launch_pdl(rmsnorm_kernel<false>, dim3((M + 7) / 8), dim3(256), 0, s, h, g, M, D, eps,
                    static_cast<void*>(u), 1.0f);
}

cudaError_t launch_rmsnorm_e4m3(const float* h, const float* g, int M, int D, float eps,
                                uint8_t* u, float oscale, cudaStream_t s) {
  return launch_pdl(rmsnorm_kernel<true>, dim3((M + 7) / 8), dim3(256), 0, s, h, g, M, D, eps,
                    static_cast<void*>(u), oscale);
}

cudaError_t launch_pixel_head(const float* F, int frames, int gh, int gw, int C, int rs,
                              int out_u8, void* pix, cudaStream_t s, int frame_rows) {
  const long long total = static_cast<long long>(C) * frames * gh * rs * gw * rs / 4;
  if (frame_rows == 0) frame_rows = gh * gw;
  return launch_pdl(pixel_head_kernel, dim3(grid_for(total, 256)), dim3(256), 0, s, F, frames,
                    frame_rows, gh, gw, C, rs, out_u8, pix);
}

cudaError_t launch_kv_append(const float* k, const float* v, int groups, int rows, int slot,
                             int ring_pitch, __nv_bfloat16* k_ring, __half* vt_ring,
                             cudaStream_t s) {
  dim3 grid((rows + 31) / 32, groups);
  return launch_pdl(kv_append_kernel, grid, dim3(32, 8), 0, s, k, v, rows, slot, ring_pitch,
                    k_ring, vt_ring);
}

cudaError_t launch_rope_table(const int* step_dev, int t_host, int nsets, const int* frames,
                              int band_t, const double* inv_freq, float2* table,
                              cudaStream_t s) {
  if (nsets < 1 || nsets > kMaxRopeSets || band_t < 1 || band_t > kRopePairs)
    return cudaErrorInvalidValue;
  RopeSets sets{};
  for (int k = 0; k < nsets; ++k) sets.frames[k] = frames[k];
  for (int i = 0; i < band_t; ++i) sets.inv_freq[i] = inv_freq[i];
  return launch_pdl(rope_table_kernel, dim3(1), dim3(128), 0, s, step_dev, t_host, nsets, band_t,
                    sets, table);
}

// One thread waits, with the decode kernels' bounded wait (mbar_wait_for) and a limit of
// limit_ns, on an mbarrier that expects one arrival that never comes: the wait gives up, ORs
// ERR_WAIT_CHECK into *err and the kernel returns. No trap, no fault; the context stays usable.
__global__ void wait_check_kernel(int* err, unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  const uint32_t b = smem_u32(&bar);
  mbar_init(b, 1);
  fence_barrier_init();
  // err may already be set by an earlier failure: then the wait gives up at once
  mbar_wait_for(b, 0, err, ERR_WAIT_CHECK, limit_ns);
}

cudaError_t launch_wait_check(int* err, unsigned long long limit_ns, cudaStream_t s) {
  wait_check_kernel<<<1, 32, 0, s>>>(err, limit_ns);
  return cudaGetLastError();
}

cudaError_t launch_advance(int* step_dev, cudaStream_t s) {
  return launch_pdl(advance_kernel, dim3(1), dim3(1), 0, s, step_dev);
}

}  // namespace fd
