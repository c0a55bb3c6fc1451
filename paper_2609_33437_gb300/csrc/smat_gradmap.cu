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

int SMAT_FAMILY(gradmap_ctas_per_sm)(int gdtype, bool pe, bool acc, int rounds) {
#define SMAT_GOCC(R, G) (pe ? (acc ? grad_occ<R, G, true, true>() : grad_occ<R, G, true, false>()) \
                           : (acc ? grad_occ<R, G, false, true>() : grad_occ<R, G, false, false>()))
  if ((rounds & 0xFF) == 7) return gdtype == DT_BF16 ? SMAT_GOCC(7 | kFamily, DT_BF16) : SMAT_GOCC(7 | kFamily, DT_F32);
  return gdtype == DT_BF16 ? SMAT_GOCC(10 | kFamily, DT_BF16) : SMAT_GOCC(10 | kFamily, DT_F32);
#undef SMAT_GOCC
}

}  // namespace smat
