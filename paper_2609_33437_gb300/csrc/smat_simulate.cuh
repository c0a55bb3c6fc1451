// Row a3 (forward) kernels, instantiated per parameter dtype by
// smat_sim_f32.cu and smat_sim_bf16.cu so the two compile in parallel.
#pragma once
#include "smat_device.cuh"

namespace smat {
namespace {

// --------------------------------------------------------------- a3: forward ---
// One 16-element group on the vector path. IDENT: c == 1 for the whole tensor
// (kept elements are theta itself); only used without per-element alpha.
// Tie elements are written as dropped and queued in tl (resolved at the end
// of the chunk); if the queue is full they are resolved here.
template <int R, int DT, int NOISE, bool PE, bool IDENT, bool J0>
__device__ __forceinline__ void sim_group16(const KArgs& a, const TView& v, const void* th_p,
                                            const void* t0_p, void* sim_p, int64_t i, uint32_t off,
                                            TieList& tl) {
  const uint64_t g0 = (uint64_t)(v.off + i);
  Raw16<DT> th, t0;
  load16<DT>(th_p, i, th);
  load16<DT>(t0_p, i, t0);
  uint32_t kw[4] = {0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u};
  if (v.flags & TF_MASK) {
    const bool tie = group_keep16<R, J0>(a, v.tid, v.t_hi, g0, kw);
    if (v.t_lo != 0u && tie && !tl.push(off >> 4)) resolve_group_ties<R, J0>(a, v.tid, v.t_hi, v.t_lo, g0, kw);
  }
  float out[16];
  const float2 c2 = splat(v.c);
  const float2 scale2 = splat(v.noise_scale);
  // noise: three blocks per group, three words per quad (see quad_fields)
  uint4 nb0 = make_uint4(0u, 0u, 0u, 0u), nb1 = nb0, nb2 = nb0;
  const uint64_t jn = 3 * (g0 >> 4);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint32_t u[4] = {0u, 0u, 0u, 0u};
    if (NOISE != NOISE_NONE) {
      if (q == 0) nb0 = stream_block<R, J0>(a, S_NOISE, v.tid, jn);
      if (q == 1) nb1 = stream_block<R, J0>(a, S_NOISE, v.tid, jn + 1);
      if (q == 2) nb2 = stream_block<R, J0>(a, S_NOISE, v.tid, jn + 2);
      if (q == 0) quad_fields(nb0.x, nb0.y, nb0.z, u);
      if (q == 1) quad_fields(nb0.w, nb1.x, nb1.y, u);
      if (q == 2) quad_fields(nb1.z, nb1.w, nb2.x, u);
      if (q == 3) quad_fields(nb2.y, nb2.z, nb2.w, u);
    }
    uint4 aw = make_uint4(0u, 0u, 0u, 0u);
    if (PE) aw = stream_block<R, J0>(a, S_ALPHA_E, v.tid, (g0 >> 2) + q);
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int e0 = 4 * q + 2 * h;  // elements e0, e0 + 1
      const float2 th2 = th.pair(e0 >> 1), t02 = t0.pair(e0 >> 1);
      float2 kv;
      if (PE) {
        const float2 cc = make_float2(__fmul_rn(alpha_elem(a, pick(aw, 2 * h)), v.inv_keep),
                                      __fmul_rn(alpha_elem(a, pick(aw, 2 * h + 1)), v.inv_keep));
        const float2 f = fma2_rn(cc, add2_rn(th2, make_float2(-t02.x, -t02.y)), t02);
        kv = make_float2(cc.x == 1.0f ? th2.x : f.x, cc.y == 1.0f ? th2.y : f.y);
      } else if (IDENT) {
        kv = th2;
      } else {
        kv = fma2_rn(c2, add2_rn(th2, make_float2(-t02.x, -t02.y)), t02);
      }
      float x0 = kept_of(kw, e0) ? kv.x : t02.x;
      float x1 = kept_of(kw, e0 + 1) ? kv.y : t02.y;
      if (NOISE != NOISE_NONE) {
        const float2 eps = noise_of2<NOISE>(u[2 * h], u[2 * h + 1], scale2);
        x0 = __fadd_rn(x0, eps.x);
        x1 = __fadd_rn(x1, eps.y);
      }
      out[e0] = x0;
      out[e0 + 1] = x1;
    }
  }
  store16<DT>(sim_p, i, out);
}

// One element given its keep decision (any alignment).
template <int R, int DT, int NOISE, bool PE>
__device__ __forceinline__ void sim_elem_as(const KArgs& a, const TView& v, const void* th_p,
                                            const void* t0_p, void* sim_p, int64_t e, bool kept) {
  const uint64_t g = (uint64_t)(v.off + e);
  float c = v.c;
  if (PE) {
    const uint4 w = stream_block<R>(a, S_ALPHA_E, v.tid, g >> 2);
    c = __fmul_rn(alpha_elem(a, pick(w, (unsigned)(g & 3))), v.inv_keep);
  }
  const float x_th = load1<DT>(th_p, e), x_t0 = load1<DT>(t0_p, e);
  float x = x_t0;
  if (kept) x = (c == 1.0f) ? x_th : __fmaf_rn(c, __fsub_rn(x_th, x_t0), x_t0);
  if (NOISE != NOISE_NONE) x = __fadd_rn(x, noise_of<NOISE>(noise_field1<R>(a, v.tid, g), v.noise_scale));
  store1<DT>(sim_p, e, x);
}

template <int R, int DT, int NOISE, bool PE, bool IDENT, bool J0>
__device__ __forceinline__ void sim_chunk(const KArgs& a, const TView& v, const DevTensor& T,
                                          const Chunk& ch) {
  const bool vec = (v.flags & TF_VEC) != 0u;
  const bool masked = (v.flags & TF_MASK) != 0u;
  TieList tl;
  for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += 16 * (int64_t)kBlock) {
    if (vec && i + 16 <= ch.end) {
      sim_group16<R, DT, NOISE, PE, IDENT, J0>(a, v, T.theta, T.theta0, T.sim, i, (uint32_t)(i - ch.begin), tl);
    } else {
      const int64_t e_end = (i + 16 < ch.end) ? i + 16 : ch.end;
      for (int64_t e = i; e < e_end; ++e) {
        const bool kept = masked ? elem_kept<R>(a, v.tid, v.t_hi, v.t_lo, (uint64_t)(v.off + e)) : true;
        sim_elem_as<R, DT, NOISE, PE>(a, v, T.theta, T.theta0, T.sim, e, kept);
      }
    }
  }
  // queued tie groups: rewrite the few elements that the low 24 bits keep
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    if (k < tl.n) {
      const int64_t gb = ch.begin + 16 * (int64_t)tl.at(k);
      uint32_t tb = group_ties16<R, J0>(a, v.tid, v.t_hi, (uint64_t)(v.off + gb));
      while (tb) {
        const int e = __ffs(tb) - 1;
        tb &= tb - 1u;
        if (tie_kept<R, J0>(a, v.tid, v.t_lo, (uint64_t)(v.off + gb + e)))
          sim_elem_as<R, DT, NOISE, PE>(a, v, T.theta, T.theta0, T.sim, gb + e, true);
      }
    }
  }
}

template <int R, int DT, int NOISE, bool PE, bool IDENT, bool J0>
__device__ __forceinline__ void sim_chunk_noise(const KArgs& a, const TView& v, const DevTensor& T,
                                                const Chunk& ch) {
  if (v.has_noise)
    sim_chunk<R, DT, NOISE, PE, IDENT, J0>(a, v, T, ch);
  else
    sim_chunk<R, DT, NOISE_NONE, PE, IDENT, J0>(a, v, T, ch);
}

// ------------------------------------------- a2 + a3 fused (sigma_rel lists) ---
// A persistent kernel that takes work items in list order from a counter:
// statistics items (a2, one chunk each) and forward items (a3). Every
// statistics item of a tensor precedes its forward items in the list (with a
// lead of about two grid widths), so the bandwidth-bound statistics of later
// tensors run beside the compute-bound forward of earlier ones. The CTA that
// finishes a tensor's last statistics chunk sums the chunk partials in chunk
// order, publishes sigma_t and releases the tensor's ready flag; forward items
// of that tensor wait for the flag.
//
// Progress: items are taken in list order and a statistics item never waits,
// so every item a waiting forward item depends on is already held by a
// running CTA. The wait is bounded all the same: after kWaitLimit polls
// (about one second) it sets bit 0 of *a.error, skips the item and returns to
// the queue.
constexpr uint32_t kWaitLimit = 1u << 22;

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ bool wait_ready(const KArgs& a, int t) {
  for (uint32_t n = 0;; ++n) {
    if (ld_acquire(a.ready + t) == a.epoch) return true;
    if (n >= kWaitLimit) {
      atomicOr(a.error, 1);
      return false;
    }
    __nanosleep(256);
  }
}

template <int R, int DT, int NOISE, bool PE>
__device__ __forceinline__ void forward_chunk(const KArgs& a, const TView& v, const DevTensor& T,
                                              const Chunk& ch) {
  const bool j0 = (uint64_t)(v.off + ch.end) <= (uint64_t(1) << 34);
  if (!PE && v.c == 1.0f) {
    if (j0) sim_chunk_noise<R, DT, NOISE, PE, true, true>(a, v, T, ch);
    else sim_chunk_noise<R, DT, NOISE, PE, true, false>(a, v, T, ch);
  } else {
    if (j0) sim_chunk_noise<R, DT, NOISE, PE, false, true>(a, v, T, ch);
    else sim_chunk_noise<R, DT, NOISE, PE, false, false>(a, v, T, ch);
  }
}

template <int R, int DT, int NOISE, bool PE>
__global__ void __launch_bounds__(kBlock, (DT == DT_BF16 && !PE) ? 3 : 2)
    stats_simulate_kernel(const __grid_constant__ KArgs a) {
  __shared__ double sh_s[kBlock / 32];
  __shared__ double sh_q[kBlock / 32];
  __shared__ int s_item;
  __shared__ int s_flag;
  for (;;) {
    if (threadIdx.x == 0) s_item = atomicAdd(a.work_counter, 1);
    __syncthreads();
    const int it = s_item;
    if (it >= a.n_items) break;  // same value in every thread
    const uint32_t code = (uint32_t)a.items[it];
    const int64_t ci = (int64_t)(code & ~kItemForward);
    const Chunk ch = a.chunks[ci];
    const DevTensor& T = a.tensors[ch.tensor];
    if (!(code & kItemForward)) {
      double ds, dq;
      chunk_delta_sums<DT>(T, ch, sh_s, sh_q, ds, dq);
      if (threadIdx.x == 0) {
        a.partials[ci].sum = ds;
        a.partials[ci].sumsq = dq;
        __threadfence();
        s_flag = (atomicAdd(a.tensor_done + ch.tensor, 1) == T.n_chunks - 1) ? 1 : 0;
      }
      __syncthreads();
      if (s_flag) {
        // last statistics chunk of this tensor: sum the partials in chunk order
        __threadfence();
        double s = 0.0, q = 0.0;
        for (int k = threadIdx.x; k < T.n_chunks; k += kBlock) {
          s += __ldcg(&a.partials[T.chunk_first + k].sum);
          q += __ldcg(&a.partials[T.chunk_first + k].sumsq);
        }
        s = warp_sum(s);
        q = warp_sum(q);
        if ((threadIdx.x & 31) == 0) {
          sh_s[threadIdx.x >> 5] = s;
          sh_q[threadIdx.x >> 5] = q;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
          double ts = 0.0, tq = 0.0;
          for (int w = 0; w < kBlock / 32; ++w) {
            ts += sh_s[w];
            tq += sh_q[w];
          }
          const float sigma = sigma_from_sums(ts, tq, T.numel, T.sigma_rel);
          a.scal[ch.tensor].sigma = sigma;
          a.scal[ch.tensor].noise_scale =
              (float)(sqrt(NOISE == NOISE_UNIFORM ? 3.0 : 2.0) * (double)sigma);
          __threadfence();
          st_release(a.ready + ch.tensor, a.epoch);
        }
      }
    } else {
      if (T.flags & TF_SIGMA_REL) {
        if (threadIdx.x == 0) s_flag = wait_ready(a, ch.tensor) ? 1 : 0;
        __syncthreads();
      } else if (threadIdx.x == 0) {
        s_flag = 1;
      }
      __syncthreads();
      if (s_flag) {
        DevScalars S;
        S.alpha = __ldcg(&a.scal[ch.tensor].alpha);
        S.c = __ldcg(&a.scal[ch.tensor].c);
        S.sigma = __ldcg(&a.scal[ch.tensor].sigma);
        S.noise_scale = __ldcg(&a.scal[ch.tensor].noise_scale);
        forward_chunk<R, DT, NOISE, PE>(a, make_view(T, S), T, ch);
      }
    }
    __syncthreads();  // s_item, s_flag and the shared sums are reused by the next item
  }
}

template <int R, int DT, int NOISE, bool PE>
__global__ void __launch_bounds__(kBlock, (DT == DT_BF16 && !PE) ? 3 : 2) simulate_kernel(const __grid_constant__ KArgs a) {
  for (int64_t ci = a.chunk_begin + blockIdx.x; ci < a.chunk_end; ci += gridDim.x) {
    const Chunk ch = a.chunks[ci];
    const DevTensor& T = a.tensors[ch.tensor];
    const TView v = make_view(T, a.scal[ch.tensor]);
    forward_chunk<R, DT, NOISE, PE>(a, v, T, ch);
  }
}


template <int R, int DT, int NOISE, bool PE>
struct FusedVariant {
  static cudaError_t run(const KArgs& a, int grid, cudaStream_t s) {
    stats_simulate_kernel<R, DT, NOISE, PE><<<grid, kBlock, 0, s>>>(a);
    return cudaGetLastError();
  }
};

template <int R, int DT>
cudaError_t fused_run(const KArgs& a, int grid, int noise, bool pe, cudaStream_t s) {
  if (noise == NOISE_GAUSSIAN)
    return pe ? FusedVariant<R, DT, NOISE_GAUSSIAN, true>::run(a, grid, s) : FusedVariant<R, DT, NOISE_GAUSSIAN, false>::run(a, grid, s);
  return pe ? FusedVariant<R, DT, NOISE_UNIFORM, true>::run(a, grid, s) : FusedVariant<R, DT, NOISE_UNIFORM, false>::run(a, grid, s);
}

template <typename Kernel>
int occupancy_of(Kernel k) {
  int v = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, k, kBlock, 0) != cudaSuccess || v < 1) v = 1;
  return v;
}

template <int R, int DT, int NOISE, bool PE>
struct SimVariant {
  static int occ() {
    static int v = occupancy_of(simulate_kernel<R, DT, NOISE, PE>);
    return v;
  }
  static cudaError_t run(const KArgs& a, int grid, cudaStream_t s) {
    simulate_kernel<R, DT, NOISE, PE><<<grid, kBlock, 0, s>>>(a);
    return cudaGetLastError();
  }
};

template <int R, int DT>
cudaError_t sim_run(const KArgs& a, int grid, int noise, bool pe, cudaStream_t s) {
  if (noise == NOISE_GAUSSIAN)
    return pe ? SimVariant<R, DT, NOISE_GAUSSIAN, true>::run(a, grid, s) : SimVariant<R, DT, NOISE_GAUSSIAN, false>::run(a, grid, s);
  return pe ? SimVariant<R, DT, NOISE_UNIFORM, true>::run(a, grid, s) : SimVariant<R, DT, NOISE_UNIFORM, false>::run(a, grid, s);
}

template <int R, int DT>
int sim_occ(int noise, bool pe) {
  if (noise == NOISE_GAUSSIAN)
    return pe ? SimVariant<R, DT, NOISE_GAUSSIAN, true>::occ() : SimVariant<R, DT, NOISE_GAUSSIAN, false>::occ();
  return pe ? SimVariant<R, DT, NOISE_UNIFORM, true>::occ() : SimVariant<R, DT, NOISE_UNIFORM, false>::occ();
}

}  // namespace
}  // namespace smat
