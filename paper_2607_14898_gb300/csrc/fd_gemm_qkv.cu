// GEMM instances for the fused QKV epilogue, on one stream or on stacked streams (the kernel
// is in fd_gemm_kernel.cuh).
#include "fd_gemm_kernel.cuh"

namespace fd {

cudaError_t launch_gemm_qkv(const CUtensorMap& tmA, const CUtensorMap& tmB,
                            const CUtensorMap& tmO, const CUtensorMap& tmK,
                            const CUtensorMap& tmV, const GemmParams& p, int bn, bool pair,
                            int num_sms, cudaStream_t s) {
  if (p.qkv.streams > 0) return launch_gemm_t<2>(tmA, tmB, tmO, tmK, tmV, p, bn, pair, num_sms, s);
  return launch_gemm_t<1>(tmA, tmB, tmO, tmK, tmV, p, bn, pair, num_sms, s);
}

}  // namespace fd
