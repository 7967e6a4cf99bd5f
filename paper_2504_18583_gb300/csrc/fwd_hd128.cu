// Persistent decode pass (fwd_kernel.cuh) for head size 128, and the
// launcher that dispatches on the head shape.
#include "fwd_kernel.cuh"

namespace pard {

cudaError_t launch_fwd_hd128(const FwdArgs& f, int group, int grid, cudaStream_t s) {
  if (group == 2) return launch_fwd_t<128, 2>(f, grid, s);
  if (group == 4) return launch_fwd_t<128, 4>(f, grid, s);
  if (group == 8) return launch_fwd_t<128, 8>(f, grid, s);
  return cudaErrorNotSupported;
}

int fwd_smem_bytes(int hd) { return hd == 128 ? FwdCfg<128>::kSmem : FwdCfg<64>::kSmem; }

cudaError_t launch_fwd(const FwdArgs& f, int hd, int group, int grid, cudaStream_t s) {
  if (hd == 128) return launch_fwd_hd128(f, group, grid, s);
  if (hd == 64) return launch_fwd_hd64(f, group, grid, s);
  return cudaErrorNotSupported;
}

}  // namespace pard
