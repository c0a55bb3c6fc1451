// Rows a2 + a3 (the persistent work-list forward, with the delta statistics of
// sigma_rel tensors) for f32 parameters. A translation unit of its own so the
// forward kernels compile in parallel.
// Compiled once per draw family (the packed layout, and with SMAT_DRAW16
// the 16-bit draw option: the _d16 launchers; smat_internal.h).
#include "smat_simulate.cuh"

namespace smat {

cudaError_t SMAT_FAMILY(launch_stats_simulate_f32)(const KArgs& a, int grid, int noise, bool per_elem_alpha,
                                                   int rounds, cudaStream_t s) {
  if (a.n_items <= 0) return cudaSuccess;
  return (rounds & 0xFF) == 7 ? fused_run<7 | kFamily, DT_F32, false>(a, grid, noise, per_elem_alpha, false, s)
                              : fused_run<10 | kFamily, DT_F32, false>(a, grid, noise, per_elem_alpha, false, s);
}

}  // namespace smat
