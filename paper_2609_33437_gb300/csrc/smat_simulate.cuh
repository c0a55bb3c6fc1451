// Row a3 (forward) kernels, instantiated per parameter dtype by
// smat_sim_f32.cu and smat_sim_bf16.cu so the two compile in parallel.
#pragma once
#include "smat_device.cuh"

namespace smat {
namespace {

// --------------------------------------------------------------- a3: forward ---
constexpr uint32_t kQueueTie = 1u;   // the group has a mask tie (low 24 bits decide)
constexpr uint32_t kQueueTail = 2u;  // the group has a Gaussian tail element

// One 16-element group on the vector path. IDENT: c == 1 for the whole tensor
// (kept elements are theta itself); only used without per-element alpha.
// Tie elements are written as dropped and Gaussian noise takes the central
// polynomial for every element; the returned flags (kQueueTie, kQueueTail)
// say whether some element needs the element path afterwards. A flagged
// group of an in-place tensor (sim == theta0) is not stored at all, since its
// theta0 is still needed; the chunk's drain recomputes it with EXACT, which
// decides ties at once and takes the full erfinv (tail included).
template <int R, int DT, int NOISE, bool PE, bool IDENT, bool J0, bool EXACT = false, bool IP = false>
__device__ __forceinline__ uint32_t sim_group16(const KArgs& a, const TView& v, const Raw16<DT>& th,
                                                const Raw16<DT>& t0, void* sim_p, int64_t i) {
  const uint64_t g0 = (uint64_t)(v.off + i);
  uint32_t kw[4] = {0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u};
  uint32_t flags = 0u;
  if (v.flags & TF_MASK) {
    const bool tie = group_keep16<R, J0>(a, v.tid, v.t_hi, g0, kw);
    if (EXACT) {
      if (v.t_lo != 0u && tie) resolve_group_ties<R, J0>(a, v.tid, v.t_hi, v.t_lo, g0, kw);
    } else {
      flags = (v.t_lo != 0u && tie) ? kQueueTie : 0u;
    }
  }
  float out[16];
  float minL = 0.0f;
  const float2 c2 = splat(v.c);
  const float2 scale2 = splat(v.noise_scale);
  // noise and per-element alpha: three blocks per group each, three words per
  // quad (see quad_fields); with 16-bit draws two blocks each, one half word
  // per element
  constexpr bool D16 = draws16<R>();
  uint4 nb0 = make_uint4(0u, 0u, 0u, 0u), nb1 = nb0, nb2 = nb0;
  uint4 ab0 = nb0, ab1 = nb0, ab2 = nb0;
  const uint64_t jn = D16 ? (g0 >> 3) : 3 * (g0 >> 4);
  if (NOISE != NOISE_NONE) {
    nb0 = stream_block<R, J0>(a, S_NOISE, v.tid, jn);
    nb1 = stream_block<R, J0>(a, S_NOISE, v.tid, jn + 1);
    if (!D16) nb2 = stream_block<R, J0>(a, S_NOISE, v.tid, jn + 2);
  }
  if (PE) {
    ab0 = stream_block<R, J0>(a, S_ALPHA_E, v.tid, jn);
    ab1 = stream_block<R, J0>(a, S_ALPHA_E, v.tid, jn + 1);
    if (!D16) ab2 = stream_block<R, J0>(a, S_ALPHA_E, v.tid, jn + 2);
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint32_t u[4] = {0u, 0u, 0u, 0u};
    if (NOISE != NOISE_NONE) {
      if (D16) {
        halves_of(q < 2 ? nb0 : nb1, q & 1, u);
      } else {
        if (q == 0) quad_fields(nb0.x, nb0.y, nb0.z, u);
        if (q == 1) quad_fields(nb0.w, nb1.x, nb1.y, u);
        if (q == 2) quad_fields(nb1.z, nb1.w, nb2.x, u);
        if (q == 3) quad_fields(nb2.y, nb2.z, nb2.w, u);
      }
    }
    uint32_t ua[4] = {0u, 0u, 0u, 0u};
    if (PE) {
      if (D16) {
        halves_of(q < 2 ? ab0 : ab1, q & 1, ua);
      } else {
        if (q == 0) quad_fields(ab0.x, ab0.y, ab0.z, ua);
        if (q == 1) quad_fields(ab0.w, ab1.x, ab1.y, ua);
        if (q == 2) quad_fields(ab1.z, ab1.w, ab2.x, ua);
        if (q == 3) quad_fields(ab2.y, ab2.z, ab2.w, ua);
      }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int e0 = 4 * q + 2 * h;  // elements e0, e0 + 1
      const float2 th2 = th.pair(e0 >> 1), t02 = t0.pair(e0 >> 1);
      float2 kv;
      if (PE) {
        const float2 cc = make_float2(__fmul_rn(alpha_of<D16>(a, ua[2 * h]), v.inv_keep),
                                      __fmul_rn(alpha_of<D16>(a, ua[2 * h + 1]), v.inv_keep));
        const float2 f = fma2_rn(cc, sub2_rn(th2, t02), t02);
        kv = make_float2(cc.x == 1.0f ? th2.x : f.x, cc.y == 1.0f ? th2.y : f.y);
      } else if (IDENT) {
        kv = th2;
      } else {
        kv = fma2_rn(c2, sub2_rn(th2, t02), t02);
      }
      float x0 = kept_of(kw, e0) ? kv.x : t02.x;
      float x1 = kept_of(kw, e0 + 1) ? kv.y : t02.y;
      if (NOISE != NOISE_NONE) {
        const float2 eps = EXACT ? noise_of2<NOISE, D16>(u[2 * h], u[2 * h + 1], scale2)
                                 : noise_group2<NOISE, D16>(u[2 * h], u[2 * h + 1], scale2, minL);
        x0 = __fadd_rn(x0, eps.x);
        x1 = __fadd_rn(x1, eps.y);
      }
      out[e0] = x0;
      out[e0 + 1] = x1;
    }
  }
  if (!EXACT && NOISE == NOISE_GAUSSIAN && minL < -8.0f) flags |= kQueueTail;
  if (!(IP && flags && (v.flags & TF_INPLACE))) store16<DT>(sim_p, i, out);
  return flags;
}

// Tail elements of the 16-element group at gidx0 (bit e set iff element e's
// L = log2(1 - x^2) < -8), computed exactly as erfinv_central2 computes L.
template <int R, bool J0>
__device__ __forceinline__ uint32_t group_tails16(const KArgs& a, uint32_t tid, uint64_t gidx0) {
  constexpr bool D16 = draws16<R>();
  const uint64_t jn = D16 ? (gidx0 >> 3) : 3 * (gidx0 >> 4);
  const uint4 b0 = stream_block<R, J0>(a, S_NOISE, tid, jn);
  const uint4 b1 = stream_block<R, J0>(a, S_NOISE, tid, jn + 1);
  const uint4 b2 = D16 ? b1 : stream_block<R, J0>(a, S_NOISE, tid, jn + 2);
  uint32_t bits = 0u;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint32_t u[4];
    if (D16) {
      halves_of(q < 2 ? b0 : b1, q & 1, u);
    } else {
      if (q == 0) quad_fields(b0.x, b0.y, b0.z, u);
      if (q == 1) quad_fields(b0.w, b1.x, b1.y, u);
      if (q == 2) quad_fields(b1.z, b1.w, b2.x, u);
      if (q == 3) quad_fields(b2.y, b2.z, b2.w, u);
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const float x = D16 ? sym16(u[r]) : sym24(u[r]);
      if (lg2_approx(__fmaf_rn(-x, x, 1.0f)) < -8.0f) bits |= 1u << (4 * q + r);
    }
  }
  return bits;
}

// One element given its keep decision (any alignment).
template <int R, int DT, int NOISE, bool PE>
__device__ __forceinline__ void sim_elem_as(const KArgs& a, const TView& v, const void* th_p,
                                            const void* t0_p, void* sim_p, int64_t e, bool kept) {
  constexpr bool D16 = draws16<R>();
  const uint64_t g = (uint64_t)(v.off + e);
  float c = v.c;
  if (PE) c = __fmul_rn(alpha_of<D16>(a, field1<R>(a, S_ALPHA_E, v.tid, g)), v.inv_keep);
  const float x_th = load1<DT>(th_p, e), x_t0 = load1<DT>(t0_p, e);
  float x = x_t0;
  if (kept) x = (c == 1.0f) ? x_th : __fmaf_rn(c, __fsub_rn(x_th, x_t0), x_t0);
  if (NOISE != NOISE_NONE) x = __fadd_rn(x, noise_of<NOISE, D16>(field1<R>(a, S_NOISE, v.tid, g), v.noise_scale));
  store1<DT>(sim_p, e, x);
}

// Rewrite the elements of a queued group that the group path got wrong: tie
// elements the low 24 bits keep, and every Gaussian tail element.
template <int R, int DT, int NOISE, bool PE, bool J0>
__device__ __forceinline__ void sim_resolve(const KArgs& a, const TView& v, const DevTensor& T, int64_t gb,
                                         uint32_t flags) {
  const uint64_t g0 = (uint64_t)(v.off + gb);
  const uint32_t tb = (flags & kQueueTie) ? group_ties16<R, J0>(a, v.tid, v.t_hi, g0) : 0u;
  const uint32_t nb = (NOISE == NOISE_GAUSSIAN && (flags & kQueueTail)) ? group_tails16<R, J0>(a, v.tid, g0) : 0u;
  const bool masked = (v.flags & TF_MASK) != 0u;
  uint32_t todo = tb | nb;
  while (todo) {
    const int e = __ffs(todo) - 1;
    todo &= todo - 1u;
    bool kept;
    if ((tb >> e) & 1u) kept = tie_kept<R, J0>(a, v.tid, v.t_lo, g0 + (uint64_t)e);
    else kept = masked ? elem_kept<R>(a, v.tid, v.t_hi, v.t_lo, g0 + (uint64_t)e) : true;
    if (kept || ((nb >> e) & 1u)) sim_elem_as<R, DT, NOISE, PE>(a, v, T.theta, T.theta0, T.sim, gb + e, kept);
  }
}

// Groups of the current chunk that need the element path, collected by all
// threads of the CTA and drained by all of them after the chunk, so the rare
// element work is spread over the whole CTA instead of serialising each
// lane's own list. Tie-only groups fill it from the front, groups with a
// Gaussian tail element from the back (one slot per group of a chunk, so it
// cannot overflow). The counters are reset by the caller before the barrier
// that precedes the chunk.
struct ChunkQueue {
  static constexpr int kGroups = kMaxChunkElems / 16;
  uint16_t e[kGroups];
  int n_tie;
  int n_tail;
};

// IP: the launch may hold in-place tensors (a separate instantiation, so the
// launches without any carry none of the in-place code).
template <int R, int DT, int NOISE, bool PE, bool IDENT, bool J0, bool IP>
__device__ __forceinline__ void sim_chunk(const KArgs& a, const TView& v, const DevTensor& T,
                                          const Chunk& ch, ChunkQueue& cq) {
  const bool vec = (v.flags & TF_VEC) != 0u;
  const bool masked = (v.flags & TF_MASK) != 0u;
  for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += 16 * (int64_t)kBlock) {
    if (vec && i + 16 <= ch.end) {
      Raw16<DT> th, t0;
      load16<DT>(T.theta, i, th);
      load16<DT>(T.theta0, i, t0);
      const uint32_t f = sim_group16<R, DT, NOISE, PE, IDENT, J0, false, IP>(a, v, th, t0, T.sim, i);
      if (f) {
        const uint32_t entry = (((uint32_t)(i - ch.begin) >> 4) << 2) | f;
        if (f & kQueueTail)
          cq.e[ChunkQueue::kGroups - 1 - atomicAdd(&cq.n_tail, 1)] = (uint16_t)entry;
        else
          cq.e[atomicAdd(&cq.n_tie, 1)] = (uint16_t)entry;
      }
    } else {
      const int64_t e_end = (i + 16 < ch.end) ? i + 16 : ch.end;
      for (int64_t e = i; e < e_end; ++e) {
        const bool kept = masked ? elem_kept<R>(a, v.tid, v.t_hi, v.t_lo, (uint64_t)(v.off + e)) : true;
        sim_elem_as<R, DT, NOISE, PE>(a, v, T.theta, T.theta0, T.sim, e, kept);
      }
    }
  }
  // the barrier also orders every thread's group stores before the rewrites
  __syncthreads();
  const int nt = cq.n_tie, nn = cq.n_tail;
  const bool inplace = IP && (v.flags & TF_INPLACE) != 0u;
#pragma unroll 1
  for (int k = threadIdx.x; k < nt + nn; k += kBlock) {
    const uint32_t q = (k < nt) ? cq.e[k] : cq.e[ChunkQueue::kGroups - nn + (k - nt)];
    const int64_t gb = ch.begin + 16 * (int64_t)(q >> 2);
    if (inplace) {
      // the group was not stored: its theta0 is intact; recompute it whole
      Raw16<DT> th, t0;
      load16<DT>(T.theta, gb, th);
      load16<DT>(T.theta0, gb, t0);
      sim_group16<R, DT, NOISE, PE, IDENT, J0, true, IP>(a, v, th, t0, T.sim, gb);
    } else {
      sim_resolve<R, DT, NOISE, PE, J0>(a, v, T, gb, q & 3u);
    }
  }
}

template <int R, int DT, int NOISE, bool PE, bool IDENT, bool J0, bool IP>
__device__ __forceinline__ void sim_chunk_noise(const KArgs& a, const TView& v, const DevTensor& T,
                                                const Chunk& ch, ChunkQueue& cq) {
  if (v.has_noise)
    sim_chunk<R, DT, NOISE, PE, IDENT, J0, IP>(a, v, T, ch, cq);
  else
    sim_chunk<R, DT, NOISE_NONE, PE, IDENT, J0, IP>(a, v, T, ch, cq);
}

// ------------------------------------------- a2 + a3 fused (sigma_rel lists) ---
// A persistent kernel that takes work items in list order from a counter:
// statistics items (a2, one chunk each) and forward items (a3). Every
// statistics item of a tensor precedes its forward items in the list (with a
// lead of about one grid width), so the bandwidth-bound statistics of later
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
__device__ __forceinline__ bool wait_ready(const KArgs& a, int t) { return wait_value(a.ready + t, a.epoch, a.error); }

// All threads of the CTA call this for the same chunk (it has a barrier).
template <int R, int DT, int NOISE, bool PE, bool IP>
__device__ __forceinline__ void forward_chunk(const KArgs& a, const TView& v, const DevTensor& T,
                                              const Chunk& ch, ChunkQueue& cq) {
  const bool j0 = (uint64_t)(v.off + ch.end) <= (uint64_t(1) << 34);
  if (!PE && v.c == 1.0f) {
    if (j0) sim_chunk_noise<R, DT, NOISE, PE, true, true, IP>(a, v, T, ch, cq);
    else sim_chunk_noise<R, DT, NOISE, PE, true, false, IP>(a, v, T, ch, cq);
  } else {
    if (j0) sim_chunk_noise<R, DT, NOISE, PE, false, true, IP>(a, v, T, ch, cq);
    else sim_chunk_noise<R, DT, NOISE, PE, false, false, IP>(a, v, T, ch, cq);
  }
}

// MINB: CTAs per SM the launch is built for. Lists with statistics items run
// the bf16 launch at four CTAs per SM (64 registers): the extra warps hide
// the statistics' memory latency (7B list: 11.98 -> 11.73 ms); forward-only
// lists keep three (80 registers, no spills in the group path).
template <int R, int DT, int NOISE, bool PE, bool IP, int MINB = ((DT == DT_BF16 && !PE) ? 3 : 2)>
__global__ void __launch_bounds__(kBlock, MINB)
    stats_simulate_kernel(const __grid_constant__ KArgs a) {
  __shared__ double sh_s[kBlock / 32];
  __shared__ double sh_q[kBlock / 32];
  __shared__ int s_item;
  __shared__ int s_flag;
  __shared__ ChunkQueue s_cq;
  for (;;) {
    if (threadIdx.x == 0) {
      s_item = atomicAdd(a.work_counter, 1);
      s_cq.n_tie = 0;
      s_cq.n_tail = 0;
    }
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
          a.scal[ch.tensor].noise_scale = noise_scale_of<NOISE>(sigma);
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
        forward_chunk<R, DT, NOISE, PE, IP>(a, make_view(T, S), T, ch, s_cq);
      }
    }
    __syncthreads();  // s_item, s_flag and the shared sums are reused by the next item
  }
}

template <int R, int DT, int NOISE, bool PE, bool IP>
__global__ void __launch_bounds__(kBlock, (DT == DT_BF16 && !PE) ? 3 : 2) simulate_kernel(const __grid_constant__ KArgs a) {
  __shared__ ChunkQueue s_cq;
  for (int64_t ci = a.chunk_begin + blockIdx.x; ci < a.chunk_end; ci += gridDim.x) {
    if (threadIdx.x == 0) {
      s_cq.n_tie = 0;
      s_cq.n_tail = 0;
    }
    __syncthreads();
    const Chunk ch = a.chunks[ci];
    const DevTensor& T = a.tensors[ch.tensor];
    const TView v = make_view(T, a.scal[ch.tensor]);
    forward_chunk<R, DT, NOISE, PE, IP>(a, v, T, ch, s_cq);
    __syncthreads();  // every thread has read the counters before the next reset
  }
}


template <typename Kernel>
int occupancy_of(Kernel k) {
  int v = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, k, kBlock, 0) != cudaSuccess || v < 1) v = 1;
  return v;
}

template <int R, int DT, int NOISE, bool PE, bool IP, int MINB = ((DT == DT_BF16 && !PE) ? 3 : 2)>
struct FusedVariant {
  static int occ() {
    static int v = occupancy_of(stats_simulate_kernel<R, DT, NOISE, PE, IP, MINB>);
    return v;
  }
  static cudaError_t run(const KArgs& a, int grid, cudaStream_t s) {
    stats_simulate_kernel<R, DT, NOISE, PE, IP, MINB><<<grid, kBlock, 0, s>>>(a);
    return cudaGetLastError();
  }
};

// wide: the list has statistics items (the four-CTA build for bf16 without
// per-element alpha and not in place; the other cases have one build).
template <int R, int DT, bool IP>
cudaError_t fused_run(const KArgs& a, int grid, int noise, bool pe, bool wide, cudaStream_t s) {
  if constexpr (DT == DT_BF16 && !IP) {
    if (wide && !pe)
      return noise == NOISE_GAUSSIAN ? FusedVariant<R, DT, NOISE_GAUSSIAN, false, IP, 4>::run(a, grid, s)
                                     : FusedVariant<R, DT, NOISE_UNIFORM, false, IP, 4>::run(a, grid, s);
  }
  if (noise == NOISE_GAUSSIAN)
    return pe ? FusedVariant<R, DT, NOISE_GAUSSIAN, true, IP>::run(a, grid, s) : FusedVariant<R, DT, NOISE_GAUSSIAN, false, IP>::run(a, grid, s);
  return pe ? FusedVariant<R, DT, NOISE_UNIFORM, true, IP>::run(a, grid, s) : FusedVariant<R, DT, NOISE_UNIFORM, false, IP>::run(a, grid, s);
}

// Resident CTAs per SM of the launch fused_run makes.
template <int R, int DT, bool IP>
int fused_occ(int noise, bool pe, bool wide) {
  if constexpr (DT == DT_BF16 && !IP) {
    if (wide && !pe)
      return noise == NOISE_GAUSSIAN ? FusedVariant<R, DT, NOISE_GAUSSIAN, false, IP, 4>::occ()
                                     : FusedVariant<R, DT, NOISE_UNIFORM, false, IP, 4>::occ();
  }
  if (noise == NOISE_GAUSSIAN)
    return pe ? FusedVariant<R, DT, NOISE_GAUSSIAN, true, IP>::occ() : FusedVariant<R, DT, NOISE_GAUSSIAN, false, IP>::occ();
  return pe ? FusedVariant<R, DT, NOISE_UNIFORM, true, IP>::occ() : FusedVariant<R, DT, NOISE_UNIFORM, false, IP>::occ();
}

template <int R, int DT, int NOISE, bool PE, bool IP>
struct SimVariant {
  static int occ() {
    static int v = occupancy_of(simulate_kernel<R, DT, NOISE, PE, IP>);
    return v;
  }
  static cudaError_t run(const KArgs& a, int grid, cudaStream_t s) {
    simulate_kernel<R, DT, NOISE, PE, IP><<<grid, kBlock, 0, s>>>(a);
    return cudaGetLastError();
  }
};

template <int R, int DT, bool IP>
cudaError_t sim_run(const KArgs& a, int grid, int noise, bool pe, cudaStream_t s) {
  if (noise == NOISE_GAUSSIAN)
    return pe ? SimVariant<R, DT, NOISE_GAUSSIAN, true, IP>::run(a, grid, s) : SimVariant<R, DT, NOISE_GAUSSIAN, false, IP>::run(a, grid, s);
  return pe ? SimVariant<R, DT, NOISE_UNIFORM, true, IP>::run(a, grid, s) : SimVariant<R, DT, NOISE_UNIFORM, false, IP>::run(a, grid, s);
}

template <int R, int DT>
int sim_occ(int noise, bool pe) {
  if (noise == NOISE_GAUSSIAN)
    return pe ? SimVariant<R, DT, NOISE_GAUSSIAN, true, false>::occ() : SimVariant<R, DT, NOISE_GAUSSIAN, false, false>::occ();
  return pe ? SimVariant<R, DT, NOISE_UNIFORM, true, false>::occ() : SimVariant<R, DT, NOISE_UNIFORM, false, false>::occ();
}

}  // namespace
}  // namespace smat
