// dc_fused_modes.cu -- instantiations of the fused kernel for the heuristic
// scorers (H2O, StreamingLLM) and for per-row budgets (rows of different
// lengths). The kernel is in dc_fused_kernel.cuh.
#include "dc_fused_kernel.cuh"

namespace dc {

cudaError_t launch_fused_heur_perrow(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                                     const FusedPolicy& fp, int num_sms, cudaStream_t s) {
  const int grid = fused_grid(p, fs, num_sms);
  // per-row budgets rank with the policy (the host keeps heuristic scorers with
  // per-row budgets on the split engine); both variants take any row length
#define DC_FUSED_LAUNCH(D, G)                                                               \
  return p.rowlen ? launch_t<D, G, true, false, false, false, true>(maps, p, st, fs, fp, grid, s) \
                  : launch_t<D, G, true, false, true>(maps, p, st, fs, fp, grid, s)
  if (p.d == 128) {
    if (p.G == 8) DC_FUSED_LAUNCH(128, 8);
    if (p.G == 4) DC_FUSED_LAUNCH(128, 4);
    if (p.G == 2) DC_FUSED_LAUNCH(128, 2);
    DC_FUSED_LAUNCH(128, 1);
  }
  if (p.G == 8) DC_FUSED_LAUNCH(64, 8);
  if (p.G == 4) DC_FUSED_LAUNCH(64, 4);
  if (p.G == 2) DC_FUSED_LAUNCH(64, 2);
  DC_FUSED_LAUNCH(64, 1);
#undef DC_FUSED_LAUNCH
}

}  // namespace dc
