// sweep_pack.cu -- the pack specializations of the body sweep (sweep_impl.cuh).
#include "sweep_impl.cuh"

namespace frk {

cudaError_t configure_sweep_pack() {
  const cudaError_t e = configure_mode<kModePack>();
  return e == cudaSuccess ? configure_mixed<kModePack>() : e;
}

cudaError_t launch_sweep_pack(uint32_t dtype, bool aligned, const SweepParams& p, int n_ctas, cudaStream_t s) {
  return launch_mode<kModePack>(dtype, aligned, p, n_ctas, s);
}

cudaError_t launch_sweep_pack_mixed(const SweepParams& p, int n_ctas, cudaStream_t s) {
  return launch_mixed<kModePack>(p, n_ctas, s);
}

cudaError_t launch_list_pack(const ListParams& p, cudaStream_t s) { return launch_list<kModePack>(p, s); }

}  // namespace frk
