// Rows a2 + a3 (the persistent work-list forward, with the delta statistics of
// sigma_rel tensors) for bf16 parameters. A translation unit of its own so the
// forward kernels compile in parallel.
// Compiled once per draw family (the packed layout, and with SMAT_DRAW16
// the 16-bit draw option: the _d16 launchers; smat_internal.h).
#include "smat_simulate.cuh"

namespace smat {

cudaError_t SMAT_FAMILY(launch_stats_simulate_bf16)(const KArgs& a, int grid, int noise, bool per_elem_alpha,
                                                    int rounds, bool wide, cudaStream_t s) {
  if (a.n_items <= 0) return cudaSuccess;
  return (rounds & 0xFF) == 7 ? fused_run<7 | kFamily, DT_BF16, false>(a, grid, noise, per_elem_alpha, wide, s)
                              : fused_run<10 | kFamily, DT_BF16, false>(a, grid, noise, per_elem_alpha, wide, s);
}

int SMAT_FAMILY(fused_wide_ctas_per_sm)(int noise, int rounds) {
  return (rounds & 0xFF) == 7 ? fused_occ<7 | kFamily, DT_BF16, false>(noise, false, true)
                              : fused_occ<10 | kFamily, DT_BF16, false>(noise, false, true);
}

}  // namespace smat
