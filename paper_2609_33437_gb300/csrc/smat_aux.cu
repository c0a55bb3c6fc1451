// Rows a1 (per-call scalars), a2 (delta statistics), a6 (mask bits) and the
// test-hook kernels, plus the launch dispatch of the forward by dtype.
#include "smat_device.cuh"

namespace smat {
namespace {

// -------------------------------------------------------- a2: delta sums ---

template <int DT>
__global__ void __launch_bounds__(kBlock) delta_stats_kernel(const __grid_constant__ KArgs a) {
  __shared__ double sh_s[kBlock / 32];
  __shared__ double sh_q[kBlock / 32];
  for (int64_t ci = a.chunk_begin + blockIdx.x; ci < a.chunk_end; ci += gridDim.x) {
    const Chunk ch = a.chunks[ci];
    const DevTensor& T = a.tensors[ch.tensor];
    if (!(T.flags & TF_SIGMA_REL)) continue;  // uniform across the CTA
    double ds, dq;
    chunk_delta_sums<DT>(T, ch, sh_s, sh_q, ds, dq);
    if (threadIdx.x == 0) {
      a.partials[ci].sum = ds;
      a.partials[ci].sumsq = dq;
    }
  }
}

// ------------------------------------------------------ a1: per-call scalars ---
template <int R, int NOISE>
__global__ void scalars_kernel(const __grid_constant__ KArgs a) {
  const int t = blockIdx.x;
  const int lane = threadIdx.x;
  const DevTensor& T = a.tensors[t];
  // reset the fused kernel's counters for the launch that follows on this stream
  if (a.tensor_done != nullptr && lane == 0) {
    a.tensor_done[t] = 0;
    if (t == 0)
      for (int r = 0; r < kMaxRanges; ++r) a.work_counter[r] = 0;
  }
  float sigma = (T.flags & TF_SIGMA_REL) ? 0.0f : T.sigma;
  if ((T.flags & TF_SIGMA_REL) && a.with_sigma) {
    double s = 0.0, q = 0.0;
    for (int k = lane; k < T.n_chunks; k += 32) {
      const StatPartial p = a.partials[T.chunk_first + k];
      s += p.sum;
      q += p.sumsq;
    }
    s = warp_sum(s);
    q = warp_sum(q);
    sigma = sigma_from_sums(s, q, T.numel, T.sigma_rel);
  }
  if (lane == 0) {
    DevScalars S;
    if (a.alpha_mode == 2) {
      S.alpha = 0.0f;
      S.c = 0.0f;
    } else {
      const uint32_t ta = (a.alpha_mode == 0) ? kGlobalAlphaTensor : T.tid;
      const uint4 w = stream_block<R>(a, S_ALPHA_T, ta, 0);
      S.alpha = alpha_elem(a, w.x);
      S.c = __fmul_rn(S.alpha, T.inv_keep);
    }
    S.sigma = sigma;
    S.noise_scale = noise_scale_of<NOISE>(sigma);
    a.scal[t] = S;
  }
}

// ------------------------------------------------------------ a6: mask bits ---
template <int R>
__global__ void __launch_bounds__(kBlock) mask_bits_kernel(const __grid_constant__ KArgs a,
                                                           int64_t numel) {
  const DevTensor& T = a.tensors[a.tensor_index];
  const int64_t nwords = (numel + 31) / 32;
  const bool masked = (T.flags & TF_MASK) != 0u;
  const bool aligned = (T.elem_offset & 15) == 0;
  for (int64_t w = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; w < nwords;
       w += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i0 = 32 * w;
    uint32_t bits = 0u;
    if (!masked) {
      bits = 0xFFFFFFFFu;
    } else if (aligned && i0 + 32 <= numel) {
      const uint64_t g0 = (uint64_t)(T.elem_offset + i0);
      uint32_t kw[4];
      for (int h = 0; h < 2; ++h) {
        if (group_keep16<R, false>(a, T.tid, T.t_hi, g0 + 16 * h, kw) && T.t_lo != 0u)
          resolve_group_ties<R, false>(a, T.tid, T.t_hi, T.t_lo, g0 + 16 * h, kw);
        for (int e = 0; e < 16; ++e) bits |= (uint32_t)kept_of(kw, e) << (16 * h + e);
      }
    } else {
      for (int k = 0; k < 32 && i0 + k < numel; ++k)
        bits |= (uint32_t)elem_kept<R>(a, T.tid, T.t_hi, T.t_lo, (uint64_t)(T.elem_offset + i0 + k)) << k;
    }
    if (i0 + 32 > numel) bits &= (1u << (numel - i0)) - 1u;
    a.bits[w] = bits;
  }
}

// ----------------------------------------------------------- Philox self-test ---
template <int R>
__global__ void debug_philox_kernel(const uint32_t* ctr, int64_t n, RoundKeys key, uint32_t k0,
                                    uint32_t k1, uint32_t* out, uint32_t* out_ref) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const uint4 c = make_uint4(ctr[4 * i], ctr[4 * i + 1], ctr[4 * i + 2], ctr[4 * i + 3]);
    const uint4 o = philox<R>(c.x, c.y, c.z, c.w, key);
    out[4 * i] = o.x;
    out[4 * i + 1] = o.y;
    out[4 * i + 2] = o.z;
    out[4 * i + 3] = o.w;
    if (out_ref != nullptr) {
      const uint4 r = curand_Philox4x32_10(c, make_uint2(k0, k1));
      out_ref[4 * i] = r.x;
      out_ref[4 * i + 1] = r.y;
      out_ref[4 * i + 2] = r.z;
      out_ref[4 * i + 3] = r.w;
    }
  }
}

// Unit noise transforms of raw words w (test hook): sym24(w >> 8) or erfinv of it.
__global__ void debug_noise_unit_kernel(const uint32_t* words, int64_t n, int noise, float* out) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const float x = sym24(words[i] >> 8);
    out[i] = (noise == NOISE_GAUSSIAN) ? erfinv_poly(x) : (noise == NOISE_LAPLACE) ? laplace_unit(x) : x;
  }
}


}  // namespace

// The launcher family (packed draws, or _d16 for the 16-bit draw option) of
// a launch is chosen here from the variant code `rounds`.
#define SMAT_BY_FAMILY(call) ((rounds & kDraw16) ? call##_d16 : call)

cudaError_t launch_simulate(const KArgs& a, int grid, int dtype, int noise, bool per_elem_alpha,
                            int rounds, bool inplace, cudaStream_t s) {
  if (noise == NOISE_LAPLACE)  // built for 10 rounds (the host refuses 7 with Laplace)
    return dtype == DT_BF16 ? SMAT_BY_FAMILY(launch_laplace_bf16)(a, grid, false, per_elem_alpha, inplace, s)
                            : SMAT_BY_FAMILY(launch_laplace_f32)(a, grid, false, per_elem_alpha, inplace, s);
  if (inplace)
    return dtype == DT_BF16 ? SMAT_BY_FAMILY(launch_simulate_inplace_bf16)(a, grid, noise, per_elem_alpha, rounds, s)
                            : SMAT_BY_FAMILY(launch_simulate_inplace_f32)(a, grid, noise, per_elem_alpha, rounds, s);
  return dtype == DT_BF16 ? SMAT_BY_FAMILY(launch_simulate_bf16)(a, grid, noise, per_elem_alpha, rounds, s)
                          : SMAT_BY_FAMILY(launch_simulate_f32)(a, grid, noise, per_elem_alpha, rounds, s);
}

cudaError_t launch_stats_simulate(const KArgs& a, int grid, int dtype, int noise, bool per_elem_alpha,
                                  int rounds, bool inplace, bool wide, cudaStream_t s) {
  if (noise == NOISE_LAPLACE)
    return dtype == DT_BF16 ? SMAT_BY_FAMILY(launch_laplace_bf16)(a, grid, true, per_elem_alpha, inplace, s)
                            : SMAT_BY_FAMILY(launch_laplace_f32)(a, grid, true, per_elem_alpha, inplace, s);
  if (inplace)
    return dtype == DT_BF16
               ? SMAT_BY_FAMILY(launch_stats_simulate_inplace_bf16)(a, grid, noise, per_elem_alpha, rounds, s)
               : SMAT_BY_FAMILY(launch_stats_simulate_inplace_f32)(a, grid, noise, per_elem_alpha, rounds, s);
  return dtype == DT_BF16 ? SMAT_BY_FAMILY(launch_stats_simulate_bf16)(a, grid, noise, per_elem_alpha, rounds, wide, s)
                          : SMAT_BY_FAMILY(launch_stats_simulate_f32)(a, grid, noise, per_elem_alpha, rounds, s);
}

int streaming_ctas_per_sm(int dtype, int noise, bool pe, int rounds) {
  return dtype == DT_BF16 ? SMAT_BY_FAMILY(simulate_ctas_per_sm_bf16)(noise, pe, rounds)
                          : SMAT_BY_FAMILY(simulate_ctas_per_sm_f32)(noise, pe, rounds);
}

int fused_wide_occ(int noise, int rounds) { return SMAT_BY_FAMILY(fused_wide_ctas_per_sm)(noise, rounds); }

cudaError_t launch_grad_map(const KArgs& a, int grid, int gdtype, bool per_elem_alpha, bool accumulate, int rounds,
                            cudaStream_t s) {
  return SMAT_BY_FAMILY(launch_gradmap)(a, grid, gdtype, per_elem_alpha, accumulate, rounds, s);
}

int grad_map_occ(int gdtype, bool per_elem_alpha, bool accumulate, int rounds) {
  return SMAT_BY_FAMILY(gradmap_ctas_per_sm)(gdtype, per_elem_alpha, accumulate, rounds);
}

cudaError_t launch_grad_map_adamw(const KArgs& a, int grid, int gdtype, int pdtype, bool per_elem_alpha, int rounds,
                                  cudaStream_t s) {
  return SMAT_BY_FAMILY(launch_gradmap_adamw)(a, grid, gdtype, pdtype, per_elem_alpha, rounds, s);
}

int grad_map_adamw_occ(int gdtype, int pdtype, bool per_elem_alpha, int rounds) {
  return SMAT_BY_FAMILY(gradmap_adamw_ctas_per_sm)(gdtype, pdtype, per_elem_alpha, rounds);
}
#undef SMAT_BY_FAMILY

cudaError_t launch_delta_stats(const KArgs& a, int grid, int dtype, cudaStream_t s) {
  if (a.chunk_end <= a.chunk_begin) return cudaSuccess;
  if (dtype == DT_BF16)
    delta_stats_kernel<DT_BF16><<<grid, kBlock, 0, s>>>(a);
  else
    delta_stats_kernel<DT_F32><<<grid, kBlock, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_scalars(const KArgs& a, int noise, int rounds, cudaStream_t s) {
  if (a.n_tensors <= 0) return cudaSuccess;
  if ((rounds & 0xFF) == 7) {  // the per-tensor Scale draw is the same in both draw families
    if (noise == NOISE_GAUSSIAN) scalars_kernel<7, NOISE_GAUSSIAN><<<a.n_tensors, 32, 0, s>>>(a);
    else if (noise == NOISE_LAPLACE) scalars_kernel<7, NOISE_LAPLACE><<<a.n_tensors, 32, 0, s>>>(a);
    else scalars_kernel<7, NOISE_UNIFORM><<<a.n_tensors, 32, 0, s>>>(a);
  } else {
    if (noise == NOISE_GAUSSIAN) scalars_kernel<10, NOISE_GAUSSIAN><<<a.n_tensors, 32, 0, s>>>(a);
    else if (noise == NOISE_LAPLACE) scalars_kernel<10, NOISE_LAPLACE><<<a.n_tensors, 32, 0, s>>>(a);
    else scalars_kernel<10, NOISE_UNIFORM><<<a.n_tensors, 32, 0, s>>>(a);
  }
  return cudaGetLastError();
}

cudaError_t launch_mask_bits(const KArgs& a, int64_t numel, int rounds, cudaStream_t s) {
  const int64_t nwords = (numel + 31) / 32;
  if (nwords <= 0) return cudaSuccess;
  int64_t blocks = (nwords + kBlock - 1) / kBlock;
  if (blocks > 65535) blocks = 65535;
  switch (rounds) {
    case 7: mask_bits_kernel<7><<<(int)blocks, kBlock, 0, s>>>(a, numel); break;
    case 7 | kDraw16: mask_bits_kernel<7 | kDraw16><<<(int)blocks, kBlock, 0, s>>>(a, numel); break;
    case 10 | kDraw16: mask_bits_kernel<10 | kDraw16><<<(int)blocks, kBlock, 0, s>>>(a, numel); break;
    default: mask_bits_kernel<10><<<(int)blocks, kBlock, 0, s>>>(a, numel); break;
  }
  return cudaGetLastError();
}

cudaError_t launch_debug_philox(const uint32_t* ctr, int64_t n, const RoundKeys& key, int rounds,
                                uint32_t* out, uint32_t* out_ref, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  int64_t blocks = (n + 127) / 128;
  if (blocks > 4096) blocks = 4096;
  if (rounds == 7)
    debug_philox_kernel<7><<<(int)blocks, 128, 0, s>>>(ctr, n, key, key.k0[0], key.k1[0], out, out_ref);
  else
    debug_philox_kernel<10><<<(int)blocks, 128, 0, s>>>(ctr, n, key, key.k0[0], key.k1[0], out, out_ref);
  return cudaGetLastError();
}

cudaError_t launch_debug_noise_unit(const uint32_t* words, int64_t n, int noise, float* out, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  int64_t blocks = (n + 255) / 256;
  if (blocks > 8192) blocks = 8192;
  debug_noise_unit_kernel<<<(int)blocks, 256, 0, s>>>(words, n, noise, out);
  return cudaGetLastError();
}

}  // namespace smat
