// dc_fused_glob.cu -- instantiations of the fused kernel for the global token
// mode (per-row partial sums) and for the full-cache comparator (attention
// only). The kernel is in dc_fused_kernel.cuh.
#include "dc_fused_kernel.cuh"

namespace dc {

cudaError_t launch_fused_glob(const FusedMaps& maps, const Dev& p, const Step& st, const FusedStep& fs,
                              const FusedPolicy& fp, int num_sms, cudaStream_t s) {
  const int grid = fused_grid(p, fs, num_sms);
  if (p.d == 128) {
    if (p.G == 8) return launch_t<128, 8, true, false, false, true>(maps, p, st, fs, fp, grid, s);
    if (p.G == 4) return launch_t<128, 4, true, false, false, true>(maps, p, st, fs, fp, grid, s);
    if (p.G == 2) return launch_t<128, 2, true, false, false, true>(maps, p, st, fs, fp, grid, s);
    return launch_t<128, 1, true, false, false, true>(maps, p, st, fs, fp, grid, s);
  }
  if (p.G == 8) return launch_t<64, 8, true, false, false, true>(maps, p, st, fs, fp, grid, s);
  if (p.G == 4) return launch_t<64, 4, true, false, false, true>(maps, p, st, fs, fp, grid, s);
  if (p.G == 2) return launch_t<64, 2, true, false, false, true>(maps, p, st, fs, fp, grid, s);
  return launch_t<64, 1, true, false, false, true>(maps, p, st, fs, fp, grid, s);
}

cudaError_t launch_fused_full(const FusedMaps& maps, const Dev& p, int n, const FusedStep& fs,
                              const FusedPolicy& fp, int num_sms, cudaStream_t s) {
  const int grid = fused_grid(p, fs, num_sms);
  Step st{};
  st.n = n;  // no previous or departing query terms: has_prev = has_dep = 0
  if (p.d == 128) {
    if (p.G == 8) return launch_t<128, 8, true, true>(maps, p, st, fs, fp, grid, s);
    if (p.G == 4) return launch_t<128, 4, true, true>(maps, p, st, fs, fp, grid, s);
    if (p.G == 2) return launch_t<128, 2, true, true>(maps, p, st, fs, fp, grid, s);
    return launch_t<128, 1, true, true>(maps, p, st, fs, fp, grid, s);
  }
  if (p.G == 8) return launch_t<64, 8, true, true>(maps, p, st, fs, fp, grid, s);
  if (p.G == 4) return launch_t<64, 4, true, true>(maps, p, st, fs, fp, grid, s);
  if (p.G == 2) return launch_t<64, 2, true, true>(maps, p, st, fs, fp, grid, s);
  return launch_t<64, 1, true, true>(maps, p, st, fs, fp, grid, s);
}

}  // namespace dc
