// dc_fused_pair.cu -- instantiations of the fused kernel on row pairs: short
// rows, one per warpgroup, so that the serial parts of one row's step (the
// statistics merge, the output, the select) overlap the other row's passes.
// The kernel is in dc_fused_kernel.cuh.
#include "dc_fused_kernel.cuh"

namespace dc {

cudaError_t launch_fused_pair(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                              const FusedPolicy& fp, int num_sms, cudaStream_t s) {
  const int pairs = p.R / 2, grid = pairs < num_sms ? pairs : num_sms;
#define DC_FUSED_LAUNCH(D, G) \
  return launch_t<D, G, false, false, false, false, false, true>(maps, p, st, fs, fp, grid, s)
  if (p.d == 128) {
    if (p.G == 4) DC_FUSED_LAUNCH(128, 4);
    if (p.G == 2) DC_FUSED_LAUNCH(128, 2);
    DC_FUSED_LAUNCH(128, 1);
  }
  if (p.G == 4) DC_FUSED_LAUNCH(64, 4);
  if (p.G == 2) DC_FUSED_LAUNCH(64, 2);
  DC_FUSED_LAUNCH(64, 1);
#undef DC_FUSED_LAUNCH
}

}  // namespace dc
