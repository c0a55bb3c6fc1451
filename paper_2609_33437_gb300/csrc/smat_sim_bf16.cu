// Row a3 (forward, grid-stride launch with SMAT_FLAG_UNFUSED_STATS) for bf16 parameters.
// Compiled once per draw family (the packed layout, and with SMAT_DRAW16
// the 16-bit draw option: the _d16 launchers; smat_internal.h).
#include "smat_simulate.cuh"

namespace smat {

cudaError_t SMAT_FAMILY(launch_simulate_bf16)(const KArgs& a, int grid, int noise, bool per_elem_alpha,
                                              int rounds, cudaStream_t s) {
  if (a.chunk_end <= a.chunk_begin) return cudaSuccess;
  return (rounds & 0xFF) == 7 ? sim_run<7 | kFamily, DT_BF16, false>(a, grid, noise, per_elem_alpha, s)
                              : sim_run<10 | kFamily, DT_BF16, false>(a, grid, noise, per_elem_alpha, s);
}

int SMAT_FAMILY(simulate_ctas_per_sm_bf16)(int noise, bool per_elem_alpha, int rounds) {
  return (rounds & 0xFF) == 7 ? sim_occ<7 | kFamily, DT_BF16>(noise, per_elem_alpha)
                              : sim_occ<10 | kFamily, DT_BF16>(noise, per_elem_alpha);
}

}  // namespace smat
