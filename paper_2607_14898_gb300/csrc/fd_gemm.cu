// GEMM instances for every epilogue but EPI_QKV, and the launch entry point (the kernel is
// in fd_gemm_kernel.cuh).
#include "fd_gemm_kernel.cuh"

namespace fd {

cudaError_t launch_gemm(const CUtensorMap& tmA, const CUtensorMap& tmB, const CUtensorMap& tmO,
                        const CUtensorMap& tmK, const CUtensorMap& tmV, const GemmParams& p,
                        int bn, bool pair, int num_sms, cudaStream_t s) {
  if (p.epi == EPI_QKV) return launch_gemm_qkv(tmA, tmB, tmO, tmK, tmV, p, bn, pair, num_sms, s);
  return launch_gemm_t<0>(tmA, tmB, tmO, tmK, tmV, p, bn, pair, num_sms, s);
}

// the scores-backward instance: tmA / tmB = Q / K, tmdO / tmV the second product's operands
cudaError_t launch_gemm_scores_bwd(const CUtensorMap& tmA, const CUtensorMap& tmB,
                                   const CUtensorMap& tmdO, const CUtensorMap& tmV,
                                   const GemmParams& p, int num_sms, cudaStream_t s) {
  return launch_bn<128, false, 0, true>(tmA, tmB, tmA, tmdO, tmV, p, num_sms, s);
}

}  // namespace fd
