// SMAT simulated-merge kernels for GB300 (sm_103a).
//
// Rows of the hot path implemented here:
//   a1 scalars_kernel      per-call scalars (Scale alpha_t, c_t = alpha_t / p_keep,
//                          sigma_t, noise scale), Sec. 4.1
//   a2 delta_stats_kernel  per-chunk sums of delta = theta - theta0 and delta^2
//   a3 simulate_kernel     theta~ = theta0 + alpha m (.) (theta - theta0) + eps
//                          (Eq. smat-state, Eq. smat-mask, Perturb of Sec. 4.1)
//   a5 gradmap_kernel      g = alpha m (.) g~ (Eq. smat-gradient), mask regenerated
//   a6 mask_bits_kernel    packed keep bits (test hook)
//
// All of them are multi-tensor launches over a chunk table: each CTA walks
// chunks of 2^16 elements of one tensor in grid-stride order; each thread
// owns 16 consecutive elements at a time (one 256-bit load per bf16 input,
// two per fp32 input), which is exactly one Philox block of the mask stream
// (16 high bytes) and four blocks of the noise stream. The random words stay
// in registers; masks and noise are never written to memory.
//
// The path is elementwise and bound by HBM bandwidth or by the integer
// pipeline (Philox): there is no contraction, so no tensor-core work.

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <curand_philox4x32_x.h>

#include "smat_internal.h"

namespace smat {
namespace {

// Philox-4x32 round multipliers (Salmon et al., SC'11).
constexpr uint32_t kMulA = 0xD2511F53u;
constexpr uint32_t kMulB = 0xCD9E8D57u;

constexpr int NOISE_UNIFORM = 0;
constexpr int NOISE_GAUSSIAN = 1;
constexpr int DT_F32 = 0;
constexpr int DT_BF16 = 1;

// One Philox-4x32-R block with round keys precomputed from the seed. Each
// round takes the full 64-bit products of words 0 and 2 with the round
// multipliers (one wide multiply each).
template <int R>
__device__ __forceinline__ uint4 philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                        const RoundKeys& k) {
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const uint64_t pA = (uint64_t)c0 * kMulA;
    const uint64_t pB = (uint64_t)c2 * kMulB;
    c0 = (uint32_t)(pB >> 32) ^ c1 ^ k.k0[r];
    c1 = (uint32_t)pB;
    c2 = (uint32_t)(pA >> 32) ^ c3 ^ k.k1[r];
    c3 = (uint32_t)pA;
  }
  return make_uint4(c0, c1, c2, c3);
}

// Block j of sub-stream `stream` of tensor `tid` at this call's step. J0: the
// caller guarantees j < 2^32, so counter word 1 is the constant 0 and the
// loop-invariant part of the first two rounds can be hoisted.
template <int R, bool J0 = false>
__device__ __forceinline__ uint4 stream_block(const KArgs& a, uint32_t stream, uint32_t tid,
                                              uint64_t j) {
  return philox<R>((uint32_t)j, J0 ? 0u : (uint32_t)(j >> 32), (stream << 28) | tid, a.step, a.key);
}

__device__ __forceinline__ uint32_t pick(const uint4& w, unsigned i) {
  return i == 0 ? w.x : (i == 1 ? w.y : (i == 2 ? w.z : w.w));
}

// u01(u) = (u >> 8) 2^-24 and sym(u) = (2 (u >> 8) + 1 - 2^24) 2^-24, both
// exact in fp32.
__device__ __forceinline__ float u01(uint32_t u) {
  return __fmul_rn(__uint2float_rn(u >> 8), 5.9604644775390625e-08f);
}
__device__ __forceinline__ float sym(uint32_t u) {
  const int k = (int)(u >> 8);
  return __fmul_rn(__int2float_rn(2 * k + 1 - (1 << 24)), 5.9604644775390625e-08f);
}

// Perturb of one element from its noise word: uniform scale * sym(n) with
// scale = fl(sqrt3 sigma), or Gaussian scale * erfinv(sym(n)) with
// scale = fl(sqrt2 sigma) (inverse-CDF transform; CUDA's erfinvf).
template <int NOISE>
__device__ __forceinline__ float noise_of(uint32_t n, float scale) {
  if (NOISE == NOISE_UNIFORM) return __fmul_rn(scale, sym(n));
  return __fmul_rn(scale, erfinvf(sym(n)));
}

// Set element e's flag without indexing kw by a run-time value (which would
// move the array to local memory).
__device__ __forceinline__ void set_kept(uint32_t (&kw)[4], int e) {
  const uint32_t bit = 0x80u << (8 * (e & 3));
  const int q = e >> 2;
  kw[0] |= (q == 0) ? bit : 0u;
  kw[1] |= (q == 1) ? bit : 0u;
  kw[2] |= (q == 2) ? bit : 0u;
  kw[3] |= (q == 3) ? bit : 0u;
}

__device__ __forceinline__ bool kept_of(const uint32_t (&kw)[4], int e) {
  return (kw[e >> 2] & (0x80u << (8 * (e & 3)))) != 0u;
}

// Keep flags of the 16 elements gidx0 .. gidx0 + 15 (gidx0 % 16 == 0). The
// high byte of each element's 32-bit mask uniform comes from one MASK block
// (byte b of word q serves element 4q + b); it is compared with the
// threshold's high byte four bytes at a time (SWAR, no carries between
// bytes). Bit 8b + 7 of kw[q] is element 4q + b's flag. Bytes equal to the
// threshold byte (probability 1/256 each) need the low 24 bits of their
// uniform from the MASK_LO stream: they are returned in *ties (bit e for
// element e, flag left clear) when ties != nullptr, else drawn here.
template <int R, bool J0>
__device__ __forceinline__ void group_keep16(const KArgs& a, uint32_t tid, uint32_t t_hi,
                                             uint32_t t_lo, uint64_t gidx0, uint32_t (&kw)[4],
                                             uint32_t* ties) {
  const uint4 w = stream_block<R, J0>(a, S_MASK, tid, gidx0 >> 4);
  const uint32_t words[4] = {w.x, w.y, w.z, w.w};
  const uint32_t tt = t_hi * 0x01010101u;
  const uint32_t tl = tt & 0x7F7F7F7Fu;
  uint32_t anytie = 0u;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint32_t x = words[q];
    // bit 7 of each byte of d: low 7 bits of x >= low 7 bits of t
    const uint32_t d = (x | 0x80808080u) - tl;
    kw[q] = ((~x & tt) | (~(x ^ tt) & ~d)) & 0x80808080u;  // x < t per byte
    const uint32_t e = x ^ tt;
    anytie |= (e - 0x01010101u) & ~e & 0x80808080u;  // nonzero iff some byte equals t
  }
  if (t_lo != 0u && anytie != 0u) {
    uint32_t tbits = 0u;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint32_t e = words[q] ^ tt;
      const uint32_t eq = ~(((e & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | e) & 0x80808080u;  // exact per byte
      tbits |= ((eq >> 7) & 1u) << (4 * q) | ((eq >> 15) & 1u) << (4 * q + 1) |
               ((eq >> 23) & 1u) << (4 * q + 2) | ((eq >> 31) & 1u) << (4 * q + 3);
    }
    if (ties != nullptr) {
      *ties = tbits;
    } else {
      while (tbits) {
        const int e = __ffs(tbits) - 1;
        tbits &= tbits - 1u;
        const uint4 l = stream_block<R, J0>(a, S_MASK_LO, tid, (gidx0 >> 2) + (uint64_t)(e >> 2));
        if ((pick(l, (unsigned)(e & 3)) >> 8) < t_lo) set_kept(kw, e);
      }
    }
  } else if (ties != nullptr) {
    *ties = 0u;
  }
}

// Tie elements whose low 24 mask bits are drawn at the end of the chunk, so
// the rare Philox call runs once for the whole warp instead of once per
// group. Up to four 16-bit in-chunk offsets per thread, two per register.
struct TieList {
  uint32_t w0 = 0u, w1 = 0u;
  int n = 0;
  __device__ __forceinline__ bool push(uint32_t off) {
    switch (n) {
      case 0: w0 = off; break;
      case 1: w0 |= off << 16; break;
      case 2: w1 = off; break;
      case 3: w1 |= off << 16; break;
      default: return false;
    }
    ++n;
    return true;
  }
  __device__ __forceinline__ uint32_t at(int k) const {
    const uint32_t w = (k < 2) ? w0 : w1;
    return (k & 1) ? (w >> 16) : (w & 0xFFFFu);
  }
};

// Low-24-bit test of one tie element.
template <int R, bool J0>
__device__ __forceinline__ bool tie_kept(const KArgs& a, uint32_t tid, uint32_t t_lo, uint64_t gidx) {
  const uint4 l = stream_block<R, J0>(a, S_MASK_LO, tid, gidx >> 2);
  return (pick(l, (unsigned)(gidx & 3)) >> 8) < t_lo;
}


// Keep decision of one element (any alignment).
template <int R>
__device__ __forceinline__ bool elem_kept(const KArgs& a, uint32_t tid, uint32_t t_hi,
                                          uint32_t t_lo, uint64_t gidx) {
  const uint4 w = stream_block<R>(a, S_MASK, tid, gidx >> 4);
  const uint32_t hi = (pick(w, (unsigned)((gidx >> 2) & 3)) >> (8u * (unsigned)(gidx & 3))) & 0xFFu;
  if (hi != t_hi) return hi < t_hi;
  if (t_lo == 0u) return false;
  const uint4 l = stream_block<R>(a, S_MASK_LO, tid, gidx >> 2);
  return (pick(l, (unsigned)(gidx & 3)) >> 8) < t_lo;
}

// ------------------------------------------------------------ memory I/O ---
__device__ __forceinline__ void ld32B(const void* p, uint32_t (&r)[8]) {
  asm("ld.global.L1::no_allocate.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7])
      : "l"(p));
}
__device__ __forceinline__ void st32B(void* p, const uint32_t (&r)[8]) {
  asm volatile("st.global.v8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "r"(r[0]), "r"(r[1]),
               "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
               : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// 16 consecutive elements starting at element i, kept as loaded (bf16: 8
// words of two elements, fp32: 16 words); 32-byte aligned under TF_VEC.
template <int DT>
struct Raw16 {
  uint32_t r[DT == DT_BF16 ? 8 : 16];
  __device__ __forceinline__ float at(int e) const {
    if (DT == DT_BF16) return __uint_as_float((e & 1) ? (r[e >> 1] & 0xFFFF0000u) : (r[e >> 1] << 16));
    return __uint_as_float(r[e]);
  }
};

template <int DT>
__device__ __forceinline__ void load16(const void* base, int64_t i, Raw16<DT>& v) {
  if (DT == DT_BF16) {
    ld32B(static_cast<const uint16_t*>(base) + i, *reinterpret_cast<uint32_t(*)[8]>(v.r));
  } else {
    const float* p = static_cast<const float*>(base) + i;
    ld32B(p, *reinterpret_cast<uint32_t(*)[8]>(v.r));
    ld32B(p + 8, *reinterpret_cast<uint32_t(*)[8]>(v.r + 8));
  }
}

template <int DT>
__device__ __forceinline__ void store16(void* base, int64_t i, const float (&v)[16]) {
  if (DT == DT_BF16) {
    uint32_t r[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) r[m] = pack_bf16x2(v[2 * m], v[2 * m + 1]);
    st32B(static_cast<uint16_t*>(base) + i, r);
  } else {
    uint32_t r[8], s[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      r[m] = __float_as_uint(v[m]);
      s[m] = __float_as_uint(v[8 + m]);
    }
    float* p = static_cast<float*>(base) + i;
    st32B(p, r);
    st32B(p + 8, s);
  }
}

template <int DT>
__device__ __forceinline__ float load1(const void* base, int64_t i) {
  if (DT == DT_BF16)
    return __uint_as_float((uint32_t)(static_cast<const uint16_t*>(base)[i]) << 16);
  return static_cast<const float*>(base)[i];
}

template <int DT>
__device__ __forceinline__ void store1(void* base, int64_t i, float v) {
  if (DT == DT_BF16) {
    const __nv_bfloat16 h = __float2bfloat16_rn(v);
    static_cast<__nv_bfloat16*>(base)[i] = h;
  } else {
    static_cast<float*>(base)[i] = v;
  }
}

__device__ __forceinline__ float alpha_elem(const KArgs& a, uint32_t u) {
  return __fmaf_rn(a.alpha_width, u01(u), a.alpha_min);
}

// Per-chunk view of one tensor's constants.
struct TView {
  int64_t off;
  uint32_t tid, flags, t_hi, t_lo;
  float inv_keep, c, noise_scale;
  bool has_noise;
};

__device__ __forceinline__ TView make_view(const DevTensor& T, const DevScalars& S) {
  TView v;
  v.off = T.elem_offset;
  v.tid = T.tid;
  v.flags = T.flags;
  v.t_hi = T.t_hi;
  v.t_lo = T.t_lo;
  v.inv_keep = T.inv_keep;
  v.c = S.c;
  v.noise_scale = S.noise_scale;
  v.has_noise = S.sigma > 0.0f;
  return v;
}

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
    uint32_t ties = 0u;
    group_keep16<R, J0>(a, v.tid, v.t_hi, v.t_lo, g0, kw, &ties);
    while (ties) {
      const int e = __ffs(ties) - 1;
      ties &= ties - 1u;
      if (!tl.push(off + (uint32_t)e) && tie_kept<R, J0>(a, v.tid, v.t_lo, g0 + (uint64_t)e))
        set_kept(kw, e);
    }
  }
  float out[16];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint4 nw = make_uint4(0u, 0u, 0u, 0u);
    if (v.has_noise) nw = stream_block<R, J0>(a, S_NOISE, v.tid, (g0 >> 2) + q);
    uint4 aw = make_uint4(0u, 0u, 0u, 0u);
    if (PE) aw = stream_block<R, J0>(a, S_ALPHA_E, v.tid, (g0 >> 2) + q);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int e = 4 * q + k;
      const float x_th = th.at(e), x_t0 = t0.at(e);
      float kept_val;
      if (PE) {
        const float c = __fmul_rn(alpha_elem(a, pick(aw, k)), v.inv_keep);
        kept_val = (c == 1.0f) ? x_th : __fmaf_rn(c, __fsub_rn(x_th, x_t0), x_t0);
      } else if (IDENT) {
        kept_val = x_th;
      } else {
        kept_val = __fmaf_rn(v.c, __fsub_rn(x_th, x_t0), x_t0);
      }
      float x = kept_of(kw, e) ? kept_val : x_t0;
      if (v.has_noise) x = __fadd_rn(x, noise_of<NOISE>(pick(nw, k), v.noise_scale));
      out[e] = x;
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
  if (v.has_noise)
    x = __fadd_rn(x, noise_of<NOISE>(pick(stream_block<R>(a, S_NOISE, v.tid, g >> 2), (unsigned)(g & 3)),
                                     v.noise_scale));
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
  // queued ties: rewrite the few that the low 24 bits keep
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    if (k < tl.n) {
      const int64_t e = ch.begin + (int64_t)tl.at(k);
      if (tie_kept<R, J0>(a, v.tid, v.t_lo, (uint64_t)(v.off + e)))
        sim_elem_as<R, DT, NOISE, PE>(a, v, T.theta, T.theta0, T.sim, e, true);
    }
  }
}

template <int R, int DT, int NOISE, bool PE>
__global__ void __launch_bounds__(kBlock, (DT == DT_BF16 && !PE) ? 4 : 2) simulate_kernel(const __grid_constant__ KArgs a) {
  for (int64_t ci = a.chunk_begin + blockIdx.x; ci < a.chunk_end; ci += gridDim.x) {
    const Chunk ch = a.chunks[ci];
    const DevTensor& T = a.tensors[ch.tensor];
    const TView v = make_view(T, a.scal[ch.tensor]);
    const bool j0 = (uint64_t)(v.off + ch.end) <= (uint64_t(1) << 34);  // gidx >> 2 < 2^32
    if (!PE && v.c == 1.0f) {
      if (j0) sim_chunk<R, DT, NOISE, PE, true, true>(a, v, T, ch);
      else sim_chunk<R, DT, NOISE, PE, true, false>(a, v, T, ch);
    } else {
      if (j0) sim_chunk<R, DT, NOISE, PE, false, true>(a, v, T, ch);
      else sim_chunk<R, DT, NOISE, PE, false, false>(a, v, T, ch);
    }
  }
}

// ---------------------------------------------------------- a5: gradient map ---
// When `defer` (no accumulation and g_out distinct from g_sim, so the
// incoming gradient can be re-read), tie elements are written as dropped (+0)
// and queued; otherwise they are resolved at once.
template <int R, int GDT, bool PE, bool ACC, bool J0>
__device__ __forceinline__ void grad_compute16(const KArgs& a, const TView& v, uint64_t g0, uint32_t off,
                                               bool defer, TieList& tl, const Raw16<GDT>& gs,
                                               const Raw16<GDT>& go, float (&out)[16]) {
  uint32_t kw[4] = {0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u};
  if (v.flags & TF_MASK) {
    if (ACC || !defer) {
      group_keep16<R, J0>(a, v.tid, v.t_hi, v.t_lo, g0, kw, nullptr);
    } else {
      uint32_t ties = 0u;
      group_keep16<R, J0>(a, v.tid, v.t_hi, v.t_lo, g0, kw, &ties);
      while (ties) {
        const int e = __ffs(ties) - 1;
        ties &= ties - 1u;
        if (!tl.push(off + (uint32_t)e) && tie_kept<R, J0>(a, v.tid, v.t_lo, g0 + (uint64_t)e))
          set_kept(kw, e);
      }
    }
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint4 aw = make_uint4(0u, 0u, 0u, 0u);
    if (PE) aw = stream_block<R, J0>(a, S_ALPHA_E, v.tid, (g0 >> 2) + q);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int e = 4 * q + k;
      const float c = PE ? __fmul_rn(alpha_elem(a, pick(aw, k)), v.inv_keep) : v.c;
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
  if (PE) {
    const uint4 w = stream_block<R>(a, S_ALPHA_E, v.tid, g >> 2);
    c = __fmul_rn(alpha_elem(a, pick(w, (unsigned)(g & 3))), v.inv_keep);
  }
  float r = kept ? __fmul_rn(c, load1<GDT>(G.g_sim, e)) : 0.0f;
  if (ACC) r = __fadd_rn(load1<GDT>(G.g_out, e), r);
  store1<GDT>(G.g_out, e, r);
}

// Two groups per iteration (strides apart) so each thread keeps two loads of
// g~ in flight before the mask work.
template <int R, int GDT, bool PE, bool ACC, bool J0>
__device__ __forceinline__ void grad_chunk(const KArgs& a, const TView& v, const GradPtr& G, const Chunk& ch) {
  constexpr int64_t kStride = 16 * (int64_t)kBlock;
  const bool masked = (v.flags & TF_MASK) != 0u;
  const bool defer = !ACC && G.g_sim != G.g_out;
  TieList tl;
  for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += 2 * kStride) {
    const int64_t i2 = i + kStride;
    if (G.vec && i2 + 16 <= ch.end) {
      Raw16<GDT> gs1, gs2, go1, go2;
      load16<GDT>(G.g_sim, i, gs1);
      load16<GDT>(G.g_sim, i2, gs2);
      if (ACC) {
        load16<GDT>(G.g_out, i, go1);
        load16<GDT>(G.g_out, i2, go2);
      }
      float out[16];
      grad_compute16<R, GDT, PE, ACC, J0>(a, v, (uint64_t)(v.off + i), (uint32_t)(i - ch.begin), defer, tl, gs1, go1, out);
      store16<GDT>(G.g_out, i, out);
      grad_compute16<R, GDT, PE, ACC, J0>(a, v, (uint64_t)(v.off + i2), (uint32_t)(i2 - ch.begin), defer, tl, gs2, go2, out);
      store16<GDT>(G.g_out, i2, out);
    } else {
      for (int half = 0; half < 2; ++half) {
        const int64_t b = half ? i2 : i;
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
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    if (k < tl.n) {
      const int64_t e = ch.begin + (int64_t)tl.at(k);
      if (tie_kept<R, J0>(a, v.tid, v.t_lo, (uint64_t)(v.off + e))) grad_elem_as<R, GDT, PE, ACC>(a, v, G, e, true);
    }
  }
}

template <int R, int GDT, bool PE, bool ACC>
__global__ void __launch_bounds__(kBlock, (GDT == DT_BF16 && !ACC) ? 3 : 2) gradmap_kernel(const __grid_constant__ KArgs a) {
  for (int64_t ci = a.chunk_begin + blockIdx.x; ci < a.chunk_end; ci += gridDim.x) {
    const Chunk ch = a.chunks[ci];
    const DevTensor& T = a.tensors[ch.tensor];
    const GradPtr G = a.grads[ch.tensor];
    const TView v = make_view(T, a.scal[ch.tensor]);
    if ((uint64_t)(v.off + ch.end) <= (uint64_t(1) << 34))
      grad_chunk<R, GDT, PE, ACC, true>(a, v, G, ch);
    else
      grad_chunk<R, GDT, PE, ACC, false>(a, v, G, ch);
  }
}

// -------------------------------------------------------- a2: delta sums ---
__device__ __forceinline__ double warp_sum(double x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
  return x;
}

template <int DT>
__global__ void __launch_bounds__(kBlock) delta_stats_kernel(const __grid_constant__ KArgs a) {
  __shared__ double sh_s[kBlock / 32];
  __shared__ double sh_q[kBlock / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int64_t ci = a.chunk_begin + blockIdx.x; ci < a.chunk_end; ci += gridDim.x) {
    const Chunk ch = a.chunks[ci];
    const DevTensor& T = a.tensors[ch.tensor];
    if (!(T.flags & TF_SIGMA_REL)) continue;  // uniform across the CTA
    const bool vec = (T.flags & TF_VEC) != 0u;
    float s = 0.0f, q = 0.0f;
    for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += 16 * (int64_t)kBlock) {
      if (vec && i + 16 <= ch.end) {
        Raw16<DT> th, t0;
        load16<DT>(T.theta, i, th);
        load16<DT>(T.theta0, i, t0);
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const float d = __fsub_rn(th.at(k), t0.at(k));
          s += d;
          q = __fmaf_rn(d, d, q);
        }
      } else {
        const int64_t e_end = (i + 16 < ch.end) ? i + 16 : ch.end;
        for (int64_t e = i; e < e_end; ++e) {
          const float d = __fsub_rn(load1<DT>(T.theta, e), load1<DT>(T.theta0, e));
          s += d;
          q = __fmaf_rn(d, d, q);
        }
      }
    }
    double ds = warp_sum((double)s), dq = warp_sum((double)q);
    if (lane == 0) {
      sh_s[warp] = ds;
      sh_q[warp] = dq;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      double ts = 0.0, tq = 0.0;
      for (int w = 0; w < kBlock / 32; ++w) {
        ts += sh_s[w];
        tq += sh_q[w];
      }
      a.partials[ci].sum = ts;
      a.partials[ci].sumsq = tq;
    }
    __syncthreads();
  }
}

// ------------------------------------------------------ a1: per-call scalars ---
template <int R, int NOISE>
__global__ void scalars_kernel(const __grid_constant__ KArgs a) {
  const int t = blockIdx.x;
  const int lane = threadIdx.x;
  const DevTensor& T = a.tensors[t];
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
    if (T.numel > 0) {
      const double n = (double)T.numel;
      const double mean = s / n;
      double var = q / n - mean * mean;
      if (var < 0.0) var = 0.0;
      sigma = (float)((double)T.sigma_rel * sqrt(var));
    } else {
      sigma = 0.0f;
    }
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
    S.noise_scale = (float)(sqrt(NOISE == NOISE_UNIFORM ? 3.0 : 2.0) * (double)sigma);
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
        group_keep16<R, false>(a, T.tid, T.t_hi, T.t_lo, g0 + 16 * h, kw, nullptr);
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

// ---------------------------------------------------------------- launchers ---
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

template <int R, int DT, int NOISE>
cudaError_t sim_pe(const KArgs& a, int grid, bool pe, cudaStream_t s) {
  return pe ? SimVariant<R, DT, NOISE, true>::run(a, grid, s)
            : SimVariant<R, DT, NOISE, false>::run(a, grid, s);
}
template <int R, int DT>
cudaError_t sim_noise(const KArgs& a, int grid, int noise, bool pe, cudaStream_t s) {
  return noise == NOISE_GAUSSIAN ? sim_pe<R, DT, NOISE_GAUSSIAN>(a, grid, pe, s)
                                 : sim_pe<R, DT, NOISE_UNIFORM>(a, grid, pe, s);
}
template <int R>
cudaError_t sim_dt(const KArgs& a, int grid, int dt, int noise, bool pe, cudaStream_t s) {
  return dt == DT_BF16 ? sim_noise<R, DT_BF16>(a, grid, noise, pe, s)
                       : sim_noise<R, DT_F32>(a, grid, noise, pe, s);
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

cudaError_t launch_simulate(const KArgs& a, int grid, int dtype, int noise, bool per_elem_alpha,
                            int rounds, cudaStream_t s) {
  if (a.chunk_end <= a.chunk_begin) return cudaSuccess;
  return rounds == 7 ? sim_dt<7>(a, grid, dtype, noise, per_elem_alpha, s)
                     : sim_dt<10>(a, grid, dtype, noise, per_elem_alpha, s);
}

cudaError_t launch_gradmap(const KArgs& a, int grid, int gdtype, bool per_elem_alpha, bool accumulate,
                           int rounds, cudaStream_t s) {
  if (a.chunk_end <= a.chunk_begin) return cudaSuccess;
  return rounds == 7 ? grad_dt<7>(a, grid, gdtype, per_elem_alpha, accumulate, s)
                     : grad_dt<10>(a, grid, gdtype, per_elem_alpha, accumulate, s);
}

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
  if (rounds == 7) {
    if (noise == NOISE_GAUSSIAN) scalars_kernel<7, NOISE_GAUSSIAN><<<a.n_tensors, 32, 0, s>>>(a);
    else scalars_kernel<7, NOISE_UNIFORM><<<a.n_tensors, 32, 0, s>>>(a);
  } else {
    if (noise == NOISE_GAUSSIAN) scalars_kernel<10, NOISE_GAUSSIAN><<<a.n_tensors, 32, 0, s>>>(a);
    else scalars_kernel<10, NOISE_UNIFORM><<<a.n_tensors, 32, 0, s>>>(a);
  }
  return cudaGetLastError();
}

cudaError_t launch_mask_bits(const KArgs& a, int64_t numel, int rounds, cudaStream_t s) {
  const int64_t nwords = (numel + 31) / 32;
  if (nwords <= 0) return cudaSuccess;
  int64_t blocks = (nwords + kBlock - 1) / kBlock;
  if (blocks > 65535) blocks = 65535;
  if (rounds == 7)
    mask_bits_kernel<7><<<(int)blocks, kBlock, 0, s>>>(a, numel);
  else
    mask_bits_kernel<10><<<(int)blocks, kBlock, 0, s>>>(a, numel);
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

int streaming_ctas_per_sm(int dtype, int noise, bool pe, int rounds) {
  // Occupancy of the forward variant in use (the gradient map uses fewer
  // registers, so the same grid keeps it resident too).
#define SMAT_OCC(R, DT, N, P) SimVariant<R, DT, N, P>::occ()
  if (rounds == 7) {
    if (dtype == DT_BF16) {
      if (noise == NOISE_GAUSSIAN) return pe ? SMAT_OCC(7, DT_BF16, NOISE_GAUSSIAN, true) : SMAT_OCC(7, DT_BF16, NOISE_GAUSSIAN, false);
      return pe ? SMAT_OCC(7, DT_BF16, NOISE_UNIFORM, true) : SMAT_OCC(7, DT_BF16, NOISE_UNIFORM, false);
    }
    if (noise == NOISE_GAUSSIAN) return pe ? SMAT_OCC(7, DT_F32, NOISE_GAUSSIAN, true) : SMAT_OCC(7, DT_F32, NOISE_GAUSSIAN, false);
    return pe ? SMAT_OCC(7, DT_F32, NOISE_UNIFORM, true) : SMAT_OCC(7, DT_F32, NOISE_UNIFORM, false);
  }
  if (dtype == DT_BF16) {
    if (noise == NOISE_GAUSSIAN) return pe ? SMAT_OCC(10, DT_BF16, NOISE_GAUSSIAN, true) : SMAT_OCC(10, DT_BF16, NOISE_GAUSSIAN, false);
    return pe ? SMAT_OCC(10, DT_BF16, NOISE_UNIFORM, true) : SMAT_OCC(10, DT_BF16, NOISE_UNIFORM, false);
  }
  if (noise == NOISE_GAUSSIAN) return pe ? SMAT_OCC(10, DT_F32, NOISE_GAUSSIAN, true) : SMAT_OCC(10, DT_F32, NOISE_GAUSSIAN, false);
  return pe ? SMAT_OCC(10, DT_F32, NOISE_UNIFORM, true) : SMAT_OCC(10, DT_F32, NOISE_UNIFORM, false);
#undef SMAT_OCC
}

int gradmap_ctas_per_sm(int gdtype, bool pe, bool acc, int rounds) {
#define SMAT_GOCC(R, G) (pe ? (acc ? grad_occ<R, G, true, true>() : grad_occ<R, G, true, false>()) \
                           : (acc ? grad_occ<R, G, false, true>() : grad_occ<R, G, false, false>()))
  if (rounds == 7) return gdtype == DT_BF16 ? SMAT_GOCC(7, DT_BF16) : SMAT_GOCC(7, DT_F32);
  return gdtype == DT_BF16 ? SMAT_GOCC(10, DT_BF16) : SMAT_GOCC(10, DT_F32);
#undef SMAT_GOCC
}

}  // namespace smat
