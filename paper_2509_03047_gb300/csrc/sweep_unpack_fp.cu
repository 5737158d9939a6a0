// sweep_unpack_fp.cu -- unpack + verify specializations of the body sweep
// (sweep_impl.cuh) that also compute the fingerprint values of the restored
// bytes, so a restore that wants both fingerprints needs no extra sweep.
#include "sweep_impl.cuh"

namespace frk {

cudaError_t configure_sweep_unpack_fp() {
  const cudaError_t e = configure_mode<kModeUnpackFp>();
  return e == cudaSuccess ? configure_mixed<kModeUnpackFp>() : e;
}

cudaError_t launch_sweep_unpack_fp(uint32_t dtype, bool aligned, const SweepParams& p, int n_ctas, cudaStream_t s) {
  return launch_mode<kModeUnpackFp>(dtype, aligned, p, n_ctas, s);
}

cudaError_t launch_sweep_unpack_fp_mixed(const SweepParams& p, int n_ctas, cudaStream_t s) {
  return launch_mixed<kModeUnpackFp>(p, n_ctas, s);
}

cudaError_t launch_list_unpack_fp(const ListParams& p, cudaStream_t s) { return launch_list<kModeUnpackFp>(p, s); }

}  // namespace frk
