// dc_fused_graph.cu -- instantiations of the fused kernel for device-counted
// steps: the step arguments advance with a counter in device memory, so that a
// CUDA-graph capture of a step replays as the following steps. The kernel is
// in dc_fused_kernel.cuh.
#include "dc_fused_kernel.cuh"

namespace dc {

cudaError_t launch_fused_graph(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                               const FusedPolicy& fp, int num_sms, cudaStream_t s) {
  // row pairs where the plain step would take them (never with half rows)
  const bool pairs = fs.half_rows == 0 && fused_pairs(p, st.n, num_sms);
  const int grid = pairs ? (p.R / 2 < num_sms ? p.R / 2 : num_sms) : fused_grid(p, fs, num_sms);
  const bool lg = st.n > fused_onchip_tokens(p.G);
#define DC_FUSED_LAUNCH(D, G)                                                                                 \
  return pairs ? launch_t<D, G, false, false, false, false, false, true, true>(maps, p, st, fs, fp, grid, s) \
         : lg  ? launch_t<D, G, true, false, false, false, false, false, true>(maps, p, st, fs, fp, grid, s) \
               : launch_t<D, G, false, false, false, false, false, false, true>(maps, p, st, fs, fp, grid, s)
  // eight query heads per KV head: never on row pairs
#define DC_FUSED_LAUNCH8(D)                                                                                   \
  return lg ? launch_t<D, 8, true, false, false, false, false, false, true>(maps, p, st, fs, fp, grid, s)    \
            : launch_t<D, 8, false, false, false, false, false, false, true>(maps, p, st, fs, fp, grid, s)
  if (p.d == 128) {
    if (p.G == 8) DC_FUSED_LAUNCH8(128);
    if (p.G == 4) DC_FUSED_LAUNCH(128, 4);
    if (p.G == 2) DC_FUSED_LAUNCH(128, 2);
    DC_FUSED_LAUNCH(128, 1);
  }
  if (p.G == 8) DC_FUSED_LAUNCH8(64);
  if (p.G == 4) DC_FUSED_LAUNCH(64, 4);
  if (p.G == 2) DC_FUSED_LAUNCH(64, 2);
  DC_FUSED_LAUNCH(64, 1);
#undef DC_FUSED_LAUNCH
#undef DC_FUSED_LAUNCH8
}

}  // namespace dc
