// Persistent decode pass (fwd_kernel.cuh) for head size 64.
#include "fwd_kernel.cuh"

namespace pard {

cudaError_t launch_fwd_hd64(const FwdArgs& f, int group, int grid, cudaStream_t s) {
  if (group == 2) return launch_fwd_t<64, 2>(f, grid, s);
  if (group == 4) return launch_fwd_t<64, 4>(f, grid, s);
  if (group == 8) return launch_fwd_t<64, 8>(f, grid, s);
  return cudaErrorNotSupported;
}

}  // namespace pard
