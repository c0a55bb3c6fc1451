// Rows a2 + a3 (work-list launch) for f32 parameters in lists with in-place
// tensors (sim == theta0): the launch of smat_fused_f32.cu instantiated
// with the in-place path (flagged groups are recomputed whole after the chunk
// instead of rewritten element by element, since their theta0 is still
// needed), so the launches of other lists carry none of its code.
// Compiled once per draw family (the packed layout, and with SMAT_DRAW16
// the 16-bit draw option: the _d16 launchers; smat_internal.h).
#include "smat_simulate.cuh"

namespace smat {

cudaError_t SMAT_FAMILY(launch_stats_simulate_inplace_f32)(const KArgs& a, int grid, int noise,
                                                           bool per_elem_alpha, int rounds, cudaStream_t s) {
  if (a.n_items <= 0) return cudaSuccess;
  return (rounds & 0xFF) == 7 ? fused_run<7 | kFamily, DT_F32, true>(a, grid, noise, per_elem_alpha, false, s)
                              : fused_run<10 | kFamily, DT_F32, true>(a, grid, noise, per_elem_alpha, false, s);
}

}  // namespace smat
