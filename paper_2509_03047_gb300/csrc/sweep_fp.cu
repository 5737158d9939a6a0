// sweep_fp.cu -- the fp specializations of the body sweep (sweep_impl.cuh).
#include "sweep_impl.cuh"

namespace frk {

cudaError_t configure_sweep_fp() { return configure_mode<kModeFingerprint>(); }

cudaError_t launch_sweep_fp(uint32_t dtype, bool aligned, const SweepParams& p, int n_ctas, cudaStream_t s) {
  return launch_mode<kModeFingerprint>(dtype, aligned, p, n_ctas, s);
}

}  // namespace frk
