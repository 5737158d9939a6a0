// sweep_fp.cu -- the fp specializations of the body sweep (sweep_impl.cuh).
#include "sweep_impl.cuh"

namespace frk {

cudaError_t configure_sweep_fp() {
  const cudaError_t e = configure_mode<kModeFingerprint>();
  return e == cudaSuccess ? configure_mixed<kModeFingerprint>() : e;
}

cudaError_t launch_sweep_fp(uint32_t dtype, bool aligned, const SweepParams& p, int n_ctas, cudaStream_t s) {
  return launch_mode<kModeFingerprint>(dtype, aligned, p, n_ctas, s);
}

cudaError_t launch_sweep_fp_mixed(const SweepParams& p, int n_ctas, cudaStream_t s) {
  return launch_mixed<kModeFingerprint>(p, n_ctas, s);
}

}  // namespace frk
