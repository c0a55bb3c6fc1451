// Row a3 (with a2 in the work-list launch) for f32 parameters with Laplace
// Perturb (Sec. 4.1, "Perturb": the matched-RMS comparison of uniform,
// Gaussian and Laplace noise), 10 Philox rounds: the forward launches
// instantiated with the Laplace transform, in a translation unit of their own.
// Compiled once per draw family (the packed layout, and with SMAT_DRAW16
// the 16-bit draw option: the _d16 launchers; smat_internal.h).
#include "smat_simulate.cuh"

namespace smat {

namespace {
template <bool PE, bool IP>
cudaError_t laplace_run(const KArgs& a, int grid, bool fused, cudaStream_t s) {
  if (fused) {
    if (a.n_items <= 0) return cudaSuccess;
    return FusedVariant<10 | kFamily, DT_F32, NOISE_LAPLACE, PE, IP>::run(a, grid, s);
  }
  if (a.chunk_end <= a.chunk_begin) return cudaSuccess;
  return SimVariant<10 | kFamily, DT_F32, NOISE_LAPLACE, PE, IP>::run(a, grid, s);
}
}  // namespace

cudaError_t SMAT_FAMILY(launch_laplace_f32)(const KArgs& a, int grid, bool fused, bool per_elem_alpha,
                                            bool inplace, cudaStream_t s) {
  if (per_elem_alpha)
    return inplace ? laplace_run<true, true>(a, grid, fused, s) : laplace_run<true, false>(a, grid, fused, s);
  return inplace ? laplace_run<false, true>(a, grid, fused, s) : laplace_run<false, false>(a, grid, fused, s);
}

}  // namespace smat
