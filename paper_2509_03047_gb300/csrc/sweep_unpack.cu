// sweep_unpack.cu -- the unpack specializations of the body sweep (sweep_impl.cuh).
#include "sweep_impl.cuh"

namespace frk {

cudaError_t configure_sweep_unpack() {
  const cudaError_t e = configure_mode<kModeUnpack>();
  return e == cudaSuccess ? configure_mixed<kModeUnpack>() : e;
}

cudaError_t launch_sweep_unpack(uint32_t dtype, bool aligned, const SweepParams& p, int n_ctas, cudaStream_t s) {
  return launch_mode<kModeUnpack>(dtype, aligned, p, n_ctas, s);
}

cudaError_t launch_sweep_unpack_mixed(const SweepParams& p, int n_ctas, cudaStream_t s) {
  return launch_mixed<kModeUnpack>(p, n_ctas, s);
}

cudaError_t launch_list_unpack(const ListParams& p, cudaStream_t s) { return launch_list<kModeUnpack>(p, s); }

}  // namespace frk
