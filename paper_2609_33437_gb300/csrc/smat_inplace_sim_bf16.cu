// Row a3 (grid-stride launch, SMAT_FLAG_UNFUSED_STATS) for bf16 parameters in
// lists with in-place tensors: the launch of smat_sim_bf16.cu instantiated with
// the in-place path (see smat_inplace_bf16.cu).
// Compiled once per draw family (the packed layout, and with SMAT_DRAW16
// the 16-bit draw option: the _d16 launchers; smat_internal.h).
#include "smat_simulate.cuh"

namespace smat {

cudaError_t SMAT_FAMILY(launch_simulate_inplace_bf16)(const KArgs& a, int grid, int noise,
                                                      bool per_elem_alpha, int rounds, cudaStream_t s) {
  if (a.chunk_end <= a.chunk_begin) return cudaSuccess;
  return (rounds & 0xFF) == 7 ? sim_run<7 | kFamily, DT_BF16, true>(a, grid, noise, per_elem_alpha, s)
                              : sim_run<10 | kFamily, DT_BF16, true>(a, grid, noise, per_elem_alpha, s);
}

}  // namespace smat
