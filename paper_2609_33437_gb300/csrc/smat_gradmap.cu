// Row a5 (gradient map) kernels and launchers.
#include "smat_device.cuh"

namespace smat {
namespace {

// ---------------------------------------------------------- a5: gradient map ---
// When `defer` (no accumulation and g_out distinct from g_sim, so the
// incoming gradient can be re-read), tie elements are written with their
// likelier outcome (kept when P(kept | tie) >= 1/2, else dropped) and the group
// is queued: the pass after the chunk rewrites only the ties that went the
// other way. Otherwise the ties are resolved at once.
template <int R, int GDT, bool PE, bool ACC, bool J0>
__device__ __forceinline__ void grad_compute16(const KArgs& a, const TView& v, uint64_t g0, uint32_t off,
                                               bool defer, TieList& tl, const Raw16<GDT>& gs,
                                               const Raw16<GDT>& go, float (&out)[16]) {
  constexpr bool D16 = draws16<R>();
  uint32_t kw[4] = {0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u};
  if (v.flags & TF_MASK) {
    if constexpr (D16) {
      group_keep16<R, J0>(a, v.tid, v.t_hi, g0, kw);  // exact 16-bit compare: no ties
    } else {
      const uint4 mb = stream_block<R, J0>(a, S_MASK, v.tid, g0 >> 4);
      const bool tie = keep_bytes16(mb, v.t_hi, kw);
      if (v.t_lo != 0u && tie) {
        if (ACC || !defer || !tl.push(off >> 4))
          resolve_block_ties<R, J0>(a, v.tid, v.t_hi, v.t_lo, mb, g0, kw);
        else if (tie_mostly_kept(v.t_lo))
          set_tie_flags(mb, v.t_hi, kw);
      }
    }
  }
  // per-element alpha: three ALPHA_E blocks per group, three words per quad;
  // with 16-bit draws two blocks, one half word per element
  uint4 ab0 = make_uint4(0u, 0u, 0u, 0u), ab1 = ab0, ab2 = ab0;
  if (PE) {
    const uint64_t jn = D16 ? (g0 >> 3) : 3 * (g0 >> 4);
    ab0 = stream_block<R, J0>(a, S_ALPHA_E, v.tid, jn);
    ab1 = stream_block<R, J0>(a, S_ALPHA_E, v.tid, jn + 1);
    if (!D16) ab2 = stream_block<R, J0>(a, S_ALPHA_E, v.tid, jn + 2);
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
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
    for (int k = 0; k < 4; ++k) {
      const int e = 4 * q + k;
      const float c = PE ? __fmul_rn(alpha_of<D16>(a, ua[k]), v.inv_keep) : v.c;
      float g = kept_of(kw, e) ? __fmul_rn(c, gs.at(e)) : 0.0f;
      if (ACC) g = __fadd_rn(go.at(e), g);
      out[e] = g;
    }
  }
}

template <int R, int GDT, bool PE, bool ACC>
__device__ __forceinline__ void grad_elem_as(const KArgs& a, const TView& v, const GradPtr& G, int64_t e,
                                             bool kept) {
  const uint64_t g = (uint64_t)(v.off + e);
  float c = v.c;
  if (PE) c = __fmul_rn(alpha_of<draws16<R>()>(a, field1<R>(a, S_ALPHA_E, v.tid, g)), v.inv_keep);
  float r = kept ? __fmul_rn(c, load1<GDT>(G.g_sim, e)) : 0.0f;
  if (ACC) r = __fadd_rn(load1<GDT>(G.g_out, e), r);
  store1<GDT>(G.g_out, e, r);
}

// Four groups per iteration (strides apart) so each thread keeps four loads
// of g~ in flight before the mask work (two: 4.39 ms, four: 4.32 ms on the
// 7B list).
template <int R, int GDT, bool PE, bool ACC, bool J0>
__device__ __forceinline__ void grad_chunk(const KArgs& a, const TView& v, const GradPtr& G, const Chunk& ch) {
  constexpr int64_t kStride = 16 * (int64_t)kBlock;
  const bool masked = (v.flags & TF_MASK) != 0u;
  const bool defer = !ACC && G.g_sim != G.g_out;
  TieList tl;
  constexpr int NG = 4;
  for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += NG * kStride) {
    if (G.vec && i + (NG - 1) * kStride + 16 <= ch.end) {
      Raw16<GDT> gs[NG], go[NG];
#pragma unroll
      for (int q = 0; q < NG; ++q) {
        load16<GDT>(G.g_sim, i + q * kStride, gs[q]);
        if (ACC) load16<GDT>(G.g_out, i + q * kStride, go[q]);
      }
#pragma unroll
      for (int q = 0; q < NG; ++q) {
        const int64_t b = i + q * kStride;
        float out[16];
        grad_compute16<R, GDT, PE, ACC, J0>(a, v, (uint64_t)(v.off + b), (uint32_t)(b - ch.begin), defer, tl, gs[q], go[q], out);
        store16<GDT>(G.g_out, b, out);
      }
    } else {
      for (int half = 0; half < NG; ++half) {
        const int64_t b = i + half * kStride;
        if (b >= ch.end) break;
        if (G.vec && b + 16 <= ch.end) {
          Raw16<GDT> gs1, go1;
          load16<GDT>(G.g_sim, b, gs1);
          if (ACC) load16<GDT>(G.g_out, b, go1);
          float out[16];
          grad_compute16<R, GDT, PE, ACC, J0>(a, v, (uint64_t)(v.off + b), (uint32_t)(b - ch.begin), defer, tl, gs1, go1, out);
          store16<GDT>(G.g_out, b, out);
        } else {
          const int64_t e_end = (b + 16 < ch.end) ? b + 16 : ch.end;
          for (int64_t e = b; e < e_end; ++e) {
            const bool kept = masked ? elem_kept<R>(a, v.tid, v.t_hi, v.t_lo, (uint64_t)(v.off + e)) : true;
            grad_elem_as<R, GDT, PE, ACC>(a, v, G, e, kept);
          }
        }
      }
    }
  }
  // Queued groups (no accumulation here): each tie element whose decision
  // differs from the outcome written for it. Rewriting a dropped tie needs no
  // read of g~, so with P(kept | tie) >= 1/2 most of these passes read nothing.
  const bool major = tie_mostly_kept(v.t_lo);
#pragma unroll 1
  for (int k = 0; k < 4; ++k) {
    if (k < tl.n) {
      const int64_t gb = ch.begin + 16 * (int64_t)tl.at(k);
      uint32_t tb = group_ties16<R, J0>(a, v.tid, v.t_hi, (uint64_t)(v.off + gb));
      uint32_t flip = 0u;
      while (tb) {
        const int e = __ffs(tb) - 1;
        tb &= tb - 1u;
        if (tie_kept<R, J0>(a, v.tid, v.t_lo, (uint64_t)(v.off + gb + e)) != major) flip |= 1u << e;
      }
      if (flip == 0u) continue;
      if (PE && !major) {
        // the group again, ties decided at once (g~ is still intact: no
        // accumulation, g_out != g_sim); cheaper than element by element,
        // where each kept tie would draw its packed alpha field again
        Raw16<GDT> gs1, go1;
        load16<GDT>(G.g_sim, gb, gs1);
        float out[16];
        TieList none;
        grad_compute16<R, GDT, PE, ACC, J0>(a, v, (uint64_t)(v.off + gb), (uint32_t)(gb - ch.begin), false, none, gs1, go1, out);
        store16<GDT>(G.g_out, gb, out);
      } else {
        while (flip) {
          const int e = __ffs(flip) - 1;
          flip &= flip - 1u;
          if (major)
            store1<GDT>(G.g_out, gb + e, 0.0f);  // dropped: +0
          else
            grad_elem_as<R, GDT, PE, ACC>(a, v, G, gb + e, true);
        }
      }
    }
  }
}

template <int R, int GDT, bool PE, bool ACC>
__global__ void __launch_bounds__(kBlock, (GDT == DT_BF16 && !ACC) ? 3 : 2) gradmap_kernel(const __grid_constant__ KArgs a) {
  const int64_t units = a.grad_units;
  for (int64_t u = units * a.chunk_begin + blockIdx.x; u < units * a.chunk_end; u += gridDim.x) {
    Chunk ch = a.chunks[u / units];
    ch.begin += (u % units) * a.grad_unit;
    if (ch.begin >= ch.end) continue;  // the tensor's last chunk is short
    if (ch.begin + a.grad_unit < ch.end) ch.end = ch.begin + a.grad_unit;
    const DevTensor& T = a.tensors[ch.tensor];
    const GradPtr G = a.grads[ch.tensor];
    const TView v = make_view(T, a.scal[ch.tensor]);
    if ((uint64_t)(v.off + ch.end) <= (uint64_t(1) << 34))
      grad_chunk<R, GDT, PE, ACC, true>(a, v, G, ch);
    else
      grad_chunk<R, GDT, PE, ACC, false>(a, v, G, ch);
  }
}


// ------------------------------------------ a5 fused with the AdamW update ---
// The gradient map followed by the optimizer's update of the original storage
// (Sec. 4.3: storage restored, theta updated with the mapped gradient). Per
// element, the gradient the map would store (Eq. smat-gradient, rounded to the
// gradient dtype; not written) drives a decoupled-weight-decay AdamW update
// of theta and the fp32 moments m1, m2, one IEEE operation at a time:
//   theta *= decay; m1 = b1 m1 + omb1 g; m2 = b2 m2 + omb2 (g g);
//   theta -= step (m1 / (sqrt(m2) / bc2 + eps))
// then theta is rounded to its dtype. One pass reads g~, theta, m1, m2 and
// writes theta, m1, m2 (22 bytes per element for bf16 theta and gradients),
// where the gradient map and a separate update move 4 + 22.
template <int GDT>
__device__ __forceinline__ float stored_grad(float g) {
  if (GDT == DT_BF16) return __bfloat162float(__float2bfloat16_rn(g));
  return g;
}

// One AdamW step in two halves: the decay and the moment updates, then the
// step along m1 / (sqrt(m2) / bc2 + eps). With ZS, zero operands skip the
// correctly rounded square root and divisions, whose general sequences are
// slow for them (the first optimizer step, where every dropped element has
// zero moments, ran at half the bandwidth without it): sqrt(+-0) = +-0,
// +-0 / bc2 = +-0 (bc2 > 0), and +-0 / den = +-0 for den > 0 (den is NaN only
// when m2 is). Both forms give the same bits.
__device__ __forceinline__ void adam_moments(const AdamScalars& o, float g, float& th, float& m1, float& m2) {
  th = __fmul_rn(th, o.decay);
  m1 = __fadd_rn(__fmul_rn(o.b1, m1), __fmul_rn(o.omb1, g));
  m2 = __fadd_rn(__fmul_rn(o.b2, m2), __fmul_rn(o.omb2, __fmul_rn(g, g)));
}

template <bool ZS>
__device__ __forceinline__ float adam_apply(const AdamScalars& o, float th, float m1, float m2) {
  if (!ZS) {
    const float den = __fadd_rn(__fdiv_rn(__fsqrt_rn(m2), o.bc2), o.eps);
    return __fsub_rn(th, __fmul_rn(o.step, __fdiv_rn(m1, den)));
  }
  float r = m2;
  if (m2 != 0.0f) r = __fdiv_rn(__fsqrt_rn(m2), o.bc2);
  const float den = __fadd_rn(r, o.eps);
  float q = m1;
  if (!(m1 == 0.0f && den > 0.0f)) q = __fdiv_rn(m1, den);
  return __fsub_rn(th, __fmul_rn(o.step, q));
}

// One 16-element group on the vector path; mask ties decided at once. All
// four operands are loaded before the mask and alpha draws, so the group's
// 192 bytes (bf16 g~ and theta) are in flight while the Philox rounds run.
template <int R, int GDT, int PDT, bool PE, bool J0>
__device__ __forceinline__ void adam_group16(const KArgs& a, const TView& v, const DevTensor& T, const AdamPtr& A,
                                             int64_t i) {
  constexpr bool D16 = draws16<R>();
  Raw16<GDT> gs;
  load16<GDT>(A.g_sim, i, gs);
  Raw16<PDT> th;
  load16<PDT>(T.theta, i, th);
  uint32_t w1[2][8], w2[2][8];
  ld32B(A.m1 + i, w1[0]);
  ld32B(A.m1 + i + 8, w1[1]);
  ld32B(A.m2 + i, w2[0]);
  ld32B(A.m2 + i + 8, w2[1]);
  const uint64_t g0 = (uint64_t)(v.off + i);
  uint32_t kw[4] = {0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u};
  if (v.flags & TF_MASK) {
    if constexpr (D16) {
      group_keep16<R, J0>(a, v.tid, v.t_hi, g0, kw);
    } else {
      const uint4 mb = stream_block<R, J0>(a, S_MASK, v.tid, g0 >> 4);
      if (keep_bytes16(mb, v.t_hi, kw) && v.t_lo != 0u) resolve_block_ties<R, J0>(a, v.tid, v.t_hi, v.t_lo, mb, g0, kw);
    }
  }
  uint4 ab0 = make_uint4(0u, 0u, 0u, 0u), ab1 = ab0, ab2 = ab0;
  if (PE) {
    const uint64_t jn = D16 ? (g0 >> 3) : 3 * (g0 >> 4);
    ab0 = stream_block<R, J0>(a, S_ALPHA_E, v.tid, jn);
    ab1 = stream_block<R, J0>(a, S_ALPHA_E, v.tid, jn + 1);
    if (!D16) ab2 = stream_block<R, J0>(a, S_ALPHA_E, v.tid, jn + 2);
  }
  float out[16];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
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
    for (int k = 0; k < 4; ++k) {
      const int e = 4 * q + k, h = e >> 3, j = e & 7;
      const float c = PE ? __fmul_rn(alpha_of<D16>(a, ua[k]), v.inv_keep) : v.c;
      const float g = kept_of(kw, e) ? stored_grad<GDT>(__fmul_rn(c, gs.at(e))) : 0.0f;
      float t = th.at(e), x1 = __uint_as_float(w1[h][j]), x2 = __uint_as_float(w2[h][j]);
      adam_moments(a.adam, g, t, x1, x2);
      out[e] = t;
      w1[h][j] = __float_as_uint(x1);
      w2[h][j] = __float_as_uint(x2);
    }
  }
  // the zero-operand form only where the warp has a zero moment (warp-uniform
  // branch: warm moments are almost never exactly zero)
  bool anyz = false;
#pragma unroll
  for (int e = 0; e < 16; ++e) anyz |= (w1[e >> 3][e & 7] << 1) == 0u || (w2[e >> 3][e & 7] << 1) == 0u;
  if (__any_sync(__activemask(), anyz)) {
#pragma unroll
    for (int e = 0; e < 16; ++e)
      out[e] = adam_apply<true>(a.adam, out[e], __uint_as_float(w1[e >> 3][e & 7]), __uint_as_float(w2[e >> 3][e & 7]));
  } else {
#pragma unroll
    for (int e = 0; e < 16; ++e)
      out[e] = adam_apply<false>(a.adam, out[e], __uint_as_float(w1[e >> 3][e & 7]), __uint_as_float(w2[e >> 3][e & 7]));
  }
  st32B(A.m1 + i, w1[0]);
  st32B(A.m1 + i + 8, w1[1]);
  st32B(A.m2 + i, w2[0]);
  st32B(A.m2 + i + 8, w2[1]);
  store16<PDT>(const_cast<void*>(T.theta), i, out);
}

template <int R, int GDT, int PDT, bool PE>
__device__ __forceinline__ void adam_elem_at(const KArgs& a, const TView& v, const DevTensor& T, const AdamPtr& A,
                                             int64_t e) {
  const uint64_t g = (uint64_t)(v.off + e);
  const bool kept = (v.flags & TF_MASK) ? elem_kept<R>(a, v.tid, v.t_hi, v.t_lo, g) : true;
  float c = v.c;
  if (PE) c = __fmul_rn(alpha_of<draws16<R>()>(a, field1<R>(a, S_ALPHA_E, v.tid, g)), v.inv_keep);
  const float gr = kept ? stored_grad<GDT>(__fmul_rn(c, load1<GDT>(A.g_sim, e))) : 0.0f;
  float t = load1<PDT>(T.theta, e), x1 = A.m1[e], x2 = A.m2[e];
  adam_moments(a.adam, gr, t, x1, x2);
  t = adam_apply<true>(a.adam, t, x1, x2);
  store1<PDT>(const_cast<void*>(T.theta), e, t);
  A.m1[e] = x1;
  A.m2[e] = x2;
}

template <int R, int GDT, int PDT, bool PE, bool J0>
__device__ __forceinline__ void adam_chunk(const KArgs& a, const TView& v, const DevTensor& T, const AdamPtr& A,
                                           const Chunk& ch) {
  for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += 16 * (int64_t)kBlock) {
    if (A.vec && i + 16 <= ch.end) {
      adam_group16<R, GDT, PDT, PE, J0>(a, v, T, A, i);
    } else {
      const int64_t e_end = (i + 16 < ch.end) ? i + 16 : ch.end;
      for (int64_t e = i; e < e_end; ++e) adam_elem_at<R, GDT, PDT, PE>(a, v, T, A, e);
    }
  }
}

template <int R, int GDT, int PDT, bool PE>
__global__ void __launch_bounds__(kBlock, 2) gradmap_adamw_kernel(const __grid_constant__ KArgs a) {
  const int64_t units = a.grad_units;
  for (int64_t u = units * a.chunk_begin + blockIdx.x; u < units * a.chunk_end; u += gridDim.x) {
    Chunk ch = a.chunks[u / units];
    ch.begin += (u % units) * a.grad_unit;
    if (ch.begin >= ch.end) continue;  // the tensor's last chunk is short
    if (ch.begin + a.grad_unit < ch.end) ch.end = ch.begin + a.grad_unit;
    const DevTensor& T = a.tensors[ch.tensor];
    const AdamPtr A = a.adams[ch.tensor];
    const TView v = make_view(T, a.scal[ch.tensor]);
    if ((uint64_t)(v.off + ch.end) <= (uint64_t(1) << 34))
      adam_chunk<R, GDT, PDT, PE, true>(a, v, T, A, ch);
    else
      adam_chunk<R, GDT, PDT, PE, false>(a, v, T, A, ch);
  }
}

template <typename Kernel>
int occupancy_of(Kernel k) {
  int v = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, k, kBlock, 0) != cudaSuccess || v < 1) v = 1;
  return v;
}

template <int R, int GDT, bool PE, bool ACC>
int grad_occ() {
  static int v = occupancy_of(gradmap_kernel<R, GDT, PE, ACC>);
  return v;
}
template <int R, int GDT, bool PE, bool ACC>
cudaError_t grad_run(const KArgs& a, int grid, cudaStream_t s) {
  gradmap_kernel<R, GDT, PE, ACC><<<grid, kBlock, 0, s>>>(a);
  return cudaGetLastError();
}
template <int R, int GDT>
cudaError_t grad_flags(const KArgs& a, int grid, bool pe, bool acc, cudaStream_t s) {
  if (pe) return acc ? grad_run<R, GDT, true, true>(a, grid, s) : grad_run<R, GDT, true, false>(a, grid, s);
  return acc ? grad_run<R, GDT, false, true>(a, grid, s) : grad_run<R, GDT, false, false>(a, grid, s);
}
template <int R>
cudaError_t grad_dt(const KArgs& a, int grid, int gdt, bool pe, bool acc, cudaStream_t s) {
  return gdt == DT_BF16 ? grad_flags<R, DT_BF16>(a, grid, pe, acc, s)
                        : grad_flags<R, DT_F32>(a, grid, pe, acc, s);
}

}  // namespace

// This translation unit is compiled once per draw family (smat_internal.h).
cudaError_t SMAT_FAMILY(launch_gradmap)(const KArgs& a, int grid, int gdtype, bool per_elem_alpha,
                                        bool accumulate, int rounds, cudaStream_t s) {
  if (a.chunk_end <= a.chunk_begin) return cudaSuccess;
  return (rounds & 0xFF) == 7 ? grad_dt<7 | kFamily>(a, grid, gdtype, per_elem_alpha, accumulate, s)
                              : grad_dt<10 | kFamily>(a, grid, gdtype, per_elem_alpha, accumulate, s);
}

namespace {
template <int R, int GDT, int PDT, bool PE>
struct AdamVariant {
  static int occ() {
    static int v = occupancy_of(gradmap_adamw_kernel<R, GDT, PDT, PE>);
    return v;
  }
  static cudaError_t run(const KArgs& a, int grid, cudaStream_t s) {
    gradmap_adamw_kernel<R, GDT, PDT, PE><<<grid, kBlock, 0, s>>>(a);
    return cudaGetLastError();
  }
};

// f(AdamVariant<R, G, P, PE>{}) for the runtime gradient dtype, parameter
// dtype and alpha mode.
template <int R, typename F>
auto adam_dispatch(int gdtype, int pdtype, bool pe, F&& f) {
  if (gdtype == DT_BF16) {
    if (pdtype == DT_BF16) return pe ? f(AdamVariant<R, DT_BF16, DT_BF16, true>{}) : f(AdamVariant<R, DT_BF16, DT_BF16, false>{});
    return pe ? f(AdamVariant<R, DT_BF16, DT_F32, true>{}) : f(AdamVariant<R, DT_BF16, DT_F32, false>{});
  }
  if (pdtype == DT_BF16) return pe ? f(AdamVariant<R, DT_F32, DT_BF16, true>{}) : f(AdamVariant<R, DT_F32, DT_BF16, false>{});
  return pe ? f(AdamVariant<R, DT_F32, DT_F32, true>{}) : f(AdamVariant<R, DT_F32, DT_F32, false>{});
}
}  // namespace

cudaError_t SMAT_FAMILY(launch_gradmap_adamw)(const KArgs& a, int grid, int gdtype, int pdtype, bool per_elem_alpha,
                                              int rounds, cudaStream_t s) {
  if (a.chunk_end <= a.chunk_begin) return cudaSuccess;
  auto run = [&](auto var) { return decltype(var)::run(a, grid, s); };
  return (rounds & 0xFF) == 7 ? adam_dispatch<7 | kFamily>(gdtype, pdtype, per_elem_alpha, run)
                              : adam_dispatch<10 | kFamily>(gdtype, pdtype, per_elem_alpha, run);
}

int SMAT_FAMILY(gradmap_adamw_ctas_per_sm)(int gdtype, int pdtype, bool per_elem_alpha, int rounds) {
  auto occ = [](auto var) { return decltype(var)::occ(); };
  return (rounds & 0xFF) == 7 ? adam_dispatch<7 | kFamily>(gdtype, pdtype, per_elem_alpha, occ)
                              : adam_dispatch<10 | kFamily>(gdtype, pdtype, per_elem_alpha, occ);
}

int SMAT_FAMILY(gradmap_ctas_per_sm)(int gdtype, bool pe, bool acc, int rounds) {
#define SMAT_GOCC(R, G) (pe ? (acc ? grad_occ<R, G, true, true>() : grad_occ<R, G, true, false>()) \
                           : (acc ? grad_occ<R, G, false, true>() : grad_occ<R, G, false, false>()))
  if ((rounds & 0xFF) == 7) return gdtype == DT_BF16 ? SMAT_GOCC(7 | kFamily, DT_BF16) : SMAT_GOCC(7 | kFamily, DT_F32);
  return gdtype == DT_BF16 ? SMAT_GOCC(10 | kFamily, DT_BF16) : SMAT_GOCC(10 | kFamily, DT_F32);
#undef SMAT_GOCC
}

}  // namespace smat
