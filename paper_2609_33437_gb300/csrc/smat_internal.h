// Internal layout shared by the host side of libsmat and its kernels.
// (The CPU oracle has its own, independent definitions.)
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

namespace smat {

// Philox sub-streams (counter word 2 = stream << 28 | tensor id).
enum : uint32_t { S_MASK = 0, S_NOISE = 1, S_ALPHA_E = 2, S_ALPHA_T = 3, S_MASK_LO = 4 };
constexpr uint32_t kGlobalAlphaTensor = 0x0FFFFFFFu;

// Elements per work chunk of the multi-tensor launches: a power of two from
// kMinChunkElems to kMaxChunkElems chosen per tensor list, about
// sqrt(64 x total elements) (the largest cs with cs^2 / 64 <= total): large
// chunks pay the per-item costs (work-list claim, descriptor loads, barriers,
// the first loads' latency) less often, many chunks keep every CTA busy to
// the end; measured best from 2^22 to 2^32 elements. Always a multiple of 16, so a chunk never
// splits a 16-element mask draw group of an aligned tensor. Statistics and
// forward work items are whole chunks; the gradient map, whose CTAs take
// its units in a fixed grid-stride order, walks units of at most
// kMaxGradUnitElems so its CTAs end closer together.
// Stream variant code passed as `rounds` to the launchers below (and the `R`
// template parameter of the kernels): the Philox rounds (10 or 7) in the low
// byte, kDraw16 set for the 16-bit draw option (see smat_device.cuh).
constexpr int kDraw16 = 0x100;

constexpr int64_t kMinChunkElems = int64_t(1) << 12;
constexpr int64_t kMaxChunkElems = int64_t(1) << 18;
constexpr int64_t kMaxGradUnitElems = int64_t(1) << 17;
constexpr int kMaxRounds = 10;

enum : uint32_t {
  TF_MASK = 1u,       // T = floor(p_keep 2^32) < 2^32: the mask stream is consulted
  TF_VEC = 2u,        // 32-byte aligned pointers and elem_offset % 16 == 0
  TF_SIGMA_REL = 4u,  // sigma_t from delta statistics
  TF_INPLACE = 8u,    // sim == theta0: the forward overwrites theta0 with theta~
};

struct DevTensor {  // 80 bytes
  const void* theta;
  const void* theta0;
  void* sim;
  int64_t numel;
  int64_t elem_offset;
  uint32_t tid;
  uint32_t flags;
  uint32_t t_hi;  // keep threshold T >> 24, in [0, 255] when TF_MASK
  uint32_t t_lo;  // T & 0xFFFFFF
  float inv_keep; // fl(1 / p_keep), 0 when p_keep == 0
  float sigma;
  float sigma_rel;
  int32_t dtype;
  int32_t chunk_first;
  int32_t n_chunks;
};

struct Chunk {  // 24 bytes
  int32_t tensor;
  int32_t pad;
  int64_t begin;  // local element range [begin, end) of the tensor
  int64_t end;
};

struct DevScalars {  // per-call scalars (row a1)
  float alpha;
  float c;
  float sigma;
  float noise_scale;
};

struct StatPartial {  // per-chunk delta sums (row a2)
  double sum;
  double sumsq;
};

struct GradPtr {
  const void* g_sim;
  void* g_out;
  uint32_t vec;  // both 32-byte aligned and elem_offset % 16 == 0
  uint32_t pad;
};

// Gradient map fused with AdamW: the incoming gradient and the fp32 moment
// buffers of one tensor (theta is the tensor's own theta).
struct AdamPtr {  // 32 bytes
  const void* g_sim;
  float* m1;
  float* m2;
  uint32_t vec;  // theta, g_sim, m1, m2 32-byte aligned and elem_offset % 16 == 0
  uint32_t pad;
};

// Per-call AdamW constants, computed in double on the host and rounded once.
struct AdamScalars {
  float decay;  // fl(1 - lr wd)
  float b1, omb1, b2, omb2;  // beta1, fl(1 - beta1), beta2, fl(1 - beta2)
  float bc2;    // fl(sqrt(1 - beta2^t))
  float step;   // fl(lr / (1 - beta1^t))
  float eps;
};

// Philox round keys, precomputed from the seed on the host.
struct RoundKeys {
  uint32_t k0[kMaxRounds];
  uint32_t k1[kMaxRounds];
};

struct KArgs {
  const DevTensor* tensors;
  const Chunk* chunks;
  DevScalars* scal;
  StatPartial* partials;
  const GradPtr* grads;
  uint32_t* bits;        // mask_bits output
  int64_t chunk_begin;   // chunk-table range handled by this launch
  int64_t chunk_end;
  int64_t grad_unit;     // gradient map: elements per unit (divides the chunk size)
  int32_t grad_units;    // gradient map: units per chunk
  RoundKeys key;
  uint32_t step;
  int32_t n_tensors;
  float alpha_min;
  float alpha_width;     // fl(alpha_max - alpha_min)
  int32_t alpha_mode;
  int32_t tensor_index;  // mask_bits: the tensor
  int32_t with_sigma;    // scalars: 1 = derive sigma_t from the delta-statistics partials
  // fused statistics + forward (stats_simulate_kernel)
  const int32_t* items;  // work items: chunk index, high bit set for a forward item
  int32_t n_items;
  int32_t* work_counter; // next item to take (zeroed by the scalars kernel)
  int32_t* tensor_done;  // statistics chunks finished per tensor (zeroed by the scalars kernel)
  uint32_t* ready;       // per tensor: epoch of the call whose sigma_t is published
  int32_t* error;        // device error flags (bit 0: a wait ran out)
  uint32_t epoch;        // this call's epoch (>= 1)
  // gradient map fused with AdamW
  const AdamPtr* adams;
  AdamScalars adam;
};

constexpr uint32_t kItemForward = 0x80000000u;
constexpr int kMaxRanges = 2;  // one item list per parameter dtype

// Kernel launchers (smat_aux.cu, smat_gradmap.cu, smat_sim_*.cu). Each
// returns the launch's error code.
cudaError_t launch_delta_stats(const KArgs& a, int grid, int dtype, cudaStream_t s);
cudaError_t launch_scalars(const KArgs& a, int noise, int rounds, cudaStream_t s);
cudaError_t launch_simulate(const KArgs& a, int grid, int dtype, int noise, bool per_elem_alpha,
                            int rounds, bool inplace, cudaStream_t s);
// wide: the list has statistics items (bf16 without per-element alpha, not
// in place, uniform or Gaussian noise: the four-CTA-per-SM build).
cudaError_t launch_stats_simulate(const KArgs& a, int grid, int dtype, int noise, bool per_elem_alpha,
                                  int rounds, bool inplace, bool wide, cudaStream_t s);
// The forward launchers below exist twice: as declared (the packed draw
// layout) and with the suffix _d16 (the 16-bit draw option). Each forward
// translation unit is compiled once per family (SMAT_DRAW16 defined for the
// second), so the default launches carry none of the option's code;
// launch_simulate and launch_stats_simulate pick the family from `rounds`.
#define SMAT_FORWARD_LAUNCHERS(sfx)                                                                           \
  cudaError_t launch_simulate_f32##sfx(const KArgs& a, int grid, int noise, bool per_elem_alpha, int rounds,   \
                                       cudaStream_t s);                                                       \
  cudaError_t launch_simulate_bf16##sfx(const KArgs& a, int grid, int noise, bool per_elem_alpha, int rounds,  \
                                        cudaStream_t s);                                                      \
  int simulate_ctas_per_sm_f32##sfx(int noise, bool per_elem_alpha, int rounds);                              \
  int simulate_ctas_per_sm_bf16##sfx(int noise, bool per_elem_alpha, int rounds);                             \
  cudaError_t launch_stats_simulate_f32##sfx(const KArgs& a, int grid, int noise, bool per_elem_alpha,        \
                                             int rounds, cudaStream_t s);                                     \
  cudaError_t launch_stats_simulate_bf16##sfx(const KArgs& a, int grid, int noise, bool per_elem_alpha,       \
                                              int rounds, bool wide, cudaStream_t s);                         \
  /* Resident CTAs per SM of the four-CTA build (bf16, uniform or Gaussian). */                              \
  int fused_wide_ctas_per_sm##sfx(int noise, int rounds);                                                     \
  /* Laplace noise (10 rounds; smat_laplace_*.cu): the work-list launch when `fused`, else the grid-stride    \
     one; in-place instantiations when `inplace`. */                                                          \
  cudaError_t launch_laplace_f32##sfx(const KArgs& a, int grid, bool fused, bool per_elem_alpha, bool inplace, \
                                      cudaStream_t s);                                                        \
  cudaError_t launch_laplace_bf16##sfx(const KArgs& a, int grid, bool fused, bool per_elem_alpha,             \
                                       bool inplace, cudaStream_t s);                                         \
  /* the same launches for lists with in-place tensors (smat_inplace_*.cu) */                                \
  cudaError_t launch_stats_simulate_inplace_f32##sfx(const KArgs& a, int grid, int noise, bool per_elem_alpha, \
                                                     int rounds, cudaStream_t s);                             \
  cudaError_t launch_stats_simulate_inplace_bf16##sfx(const KArgs& a, int grid, int noise,                    \
                                                      bool per_elem_alpha, int rounds, cudaStream_t s);       \
  cudaError_t launch_simulate_inplace_f32##sfx(const KArgs& a, int grid, int noise, bool per_elem_alpha,      \
                                               int rounds, cudaStream_t s);                                   \
  cudaError_t launch_simulate_inplace_bf16##sfx(const KArgs& a, int grid, int noise, bool per_elem_alpha,     \
                                                int rounds, cudaStream_t s);                                  \
  cudaError_t launch_gradmap##sfx(const KArgs& a, int grid, int gdtype, bool per_elem_alpha, bool accumulate, \
                                  int rounds, cudaStream_t s);                                                \
  int gradmap_ctas_per_sm##sfx(int gdtype, bool per_elem_alpha, bool accumulate, int rounds);                 \
  cudaError_t launch_gradmap_adamw##sfx(const KArgs& a, int grid, int gdtype, int pdtype, bool per_elem_alpha, \
                                        int rounds, cudaStream_t s);                                          \
  int gradmap_adamw_ctas_per_sm##sfx(int gdtype, int pdtype, bool per_elem_alpha, int rounds);
SMAT_FORWARD_LAUNCHERS()
SMAT_FORWARD_LAUNCHERS(_d16)
#undef SMAT_FORWARD_LAUNCHERS

// Family dispatch (smat_aux.cu): the four-CTA build's occupancy and the
// gradient map for the variant code `rounds`.
int fused_wide_occ(int noise, int rounds);
cudaError_t launch_grad_map(const KArgs& a, int grid, int gdtype, bool per_elem_alpha, bool accumulate, int rounds,
                            cudaStream_t s);
int grad_map_occ(int gdtype, bool per_elem_alpha, bool accumulate, int rounds);
cudaError_t launch_grad_map_adamw(const KArgs& a, int grid, int gdtype, int pdtype, bool per_elem_alpha, int rounds,
                                  cudaStream_t s);
int grad_map_adamw_occ(int gdtype, int pdtype, bool per_elem_alpha, int rounds);

// In the forward and gradient-map translation units: the family being
// compiled (see above) and the name of its launchers.
#ifdef SMAT_DRAW16
#define SMAT_FAMILY(name) name##_d16
constexpr int kFamily = kDraw16;
#else
#define SMAT_FAMILY(name) name
constexpr int kFamily = 0;
#endif
cudaError_t launch_mask_bits(const KArgs& a, int64_t numel, int rounds, cudaStream_t s);
cudaError_t launch_debug_philox(const uint32_t* ctr, int64_t n, const RoundKeys& key, int rounds,
                                uint32_t* out, uint32_t* out_ref, cudaStream_t s);
cudaError_t launch_debug_noise_unit(const uint32_t* words, int64_t n, int noise, float* out, cudaStream_t s);
// Resident CTAs per SM of the streaming kernels (for grid sizing).
int streaming_ctas_per_sm(int dtype, int noise, bool per_elem_alpha, int rounds);

constexpr int kBlock = 256;

// Record `msg` as this thread's smat_last_error() text; returns `status`.
int record_error_code(int status, const char* msg);
// 1 if kernels can dereference p as it is, 0 if not, -1 on a CUDA error.
int gpu_can_access(const void* p);
// Philox round keys of a seed (smat_host.cpp).
RoundKeys make_round_keys(uint64_t seed);

}  // namespace smat
