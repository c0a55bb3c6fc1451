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

// One Philox-4x32-R block with round keys precomputed from the seed.
template <int R>
__device__ __forceinline__ uint4 philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                        const RoundKeys& k) {
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const uint32_t hiA = __umulhi(kMulA, c0);
    const uint32_t loA = kMulA * c0;
    const uint32_t hiB = __umulhi(kMulB, c2);
    const uint32_t loB = kMulB * c2;
    c0 = hiB ^ c1 ^ k.k0[r];
    c1 = loB;
    c2 = hiA ^ c3 ^ k.k1[r];
    c3 = loA;
  }
  return make_uint4(c0, c1, c2, c3);
}

// Block j of sub-stream `stream` of tensor `tid` at this call's step.
template <int R>
__device__ __forceinline__ uint4 stream_block(const KArgs& a, uint32_t stream, uint32_t tid,
                                              uint64_t j) {
  return philox<R>((uint32_t)j, (uint32_t)(j >> 32), (stream << 28) | tid, a.step, a.key);
}

__device__ __forceinline__ uint32_t pick(const uint4& w, unsigned i) {
  return i == 0 ? w.x : (i == 1 ? w.y : (i == 2 ? w.z : w.w));
}

// u01(u) = (u >> 8) 2^-24, u01_open(u) = ((u >> 8) + 1) 2^-24,
// sym(u) = (2 (u >> 8) + 1 - 2^24) 2^-24; all exact in fp32.
__device__ __forceinline__ float u01(uint32_t u) {
  return __fmul_rn(__uint2float_rn(u >> 8), 5.9604644775390625e-08f);
}
__device__ __forceinline__ float u01_open(uint32_t u) {
  return __fmul_rn(__uint2float_rn((u >> 8) + 1u), 5.9604644775390625e-08f);
}
__device__ __forceinline__ float sym(uint32_t u) {
  const int k = (int)(u >> 8);
  return __fmul_rn(__int2float_rn(2 * k + 1 - (1 << 24)), 5.9604644775390625e-08f);
}

// Standard-normal pair from two words (Box-Muller; CUDA's logf / sqrtf /
// sincospif, 2 u01(b) is exact so the angle needs no reduction).
__device__ __forceinline__ void box_muller(uint32_t a, uint32_t b, float& z0, float& z1) {
  const float rho = sqrtf(__fmul_rn(-2.0f, logf(u01_open(a))));
  float s, c;
  sincospif(__fmul_rn(2.0f, u01(b)), &s, &c);
  z0 = __fmul_rn(rho, c);
  z1 = __fmul_rn(rho, s);
}

template <int NOISE>
__device__ __forceinline__ void noise4(const uint4& w, float scale, float (&eps)[4]) {
  if (NOISE == NOISE_UNIFORM) {
    eps[0] = __fmul_rn(scale, sym(w.x));
    eps[1] = __fmul_rn(scale, sym(w.y));
    eps[2] = __fmul_rn(scale, sym(w.z));
    eps[3] = __fmul_rn(scale, sym(w.w));
  } else {
    float z0, z1, z2, z3;
    box_muller(w.x, w.y, z0, z1);
    box_muller(w.z, w.w, z2, z3);
    eps[0] = __fmul_rn(scale, z0);
    eps[1] = __fmul_rn(scale, z1);
    eps[2] = __fmul_rn(scale, z2);
    eps[3] = __fmul_rn(scale, z3);
  }
}

template <int NOISE>
__device__ __forceinline__ float noise1(const uint4& w, unsigned word, float scale) {
  if (NOISE == NOISE_UNIFORM) return __fmul_rn(scale, sym(pick(w, word)));
  float z0, z1;
  if (word < 2)
    box_muller(w.x, w.y, z0, z1);
  else
    box_muller(w.z, w.w, z0, z1);
  return __fmul_rn(scale, (word & 1u) ? z1 : z0);
}

// Keep bits of the 16 elements gidx0 .. gidx0 + 15 (gidx0 % 16 == 0): the high
// byte of each element's mask uniform comes from one MASK block; the low 24
// bits are drawn only when the byte ties with the threshold's high byte.
template <int R>
__device__ __forceinline__ uint32_t group_keep16(const KArgs& a, uint32_t tid, uint32_t t_hi,
                                                 uint32_t t_lo, uint64_t gidx0) {
  const uint4 w = stream_block<R>(a, S_MASK, tid, gidx0 >> 4);
  const uint32_t words[4] = {w.x, w.y, w.z, w.w};
  uint32_t keep = 0u, tie = 0u;
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const uint32_t hi = (words[k >> 2] >> (8 * (k & 3))) & 0xFFu;
    keep |= (uint32_t)(hi < t_hi) << k;
    tie |= (uint32_t)(hi == t_hi) << k;
  }
  if (t_lo == 0u) tie = 0u;  // U = T_hi 2^24 + lo >= T: dropped without a draw
  while (tie) {
    const int k = __ffs(tie) - 1;
    tie &= tie - 1u;
    const uint4 l = stream_block<R>(a, S_MASK_LO, tid, (gidx0 >> 2) + (uint64_t)(k >> 2));
    keep |= (uint32_t)((pick(l, k & 3) >> 8) < t_lo) << k;
  }
  return keep;
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

// 16 consecutive elements starting at element i (32-byte aligned for bf16,
// 64-byte aligned for fp32 under TF_VEC), widened to fp32.
template <int DT>
__device__ __forceinline__ void load16(const void* base, int64_t i, float (&v)[16]) {
  if (DT == DT_BF16) {
    uint32_t r[8];
    ld32B(static_cast<const uint16_t*>(base) + i, r);
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      v[2 * m] = __uint_as_float(r[m] << 16);
      v[2 * m + 1] = __uint_as_float(r[m] & 0xFFFF0000u);
    }
  } else {
    uint32_t r[8], s[8];
    const float* p = static_cast<const float*>(base) + i;
    ld32B(p, r);
    ld32B(p + 8, s);
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      v[m] = __uint_as_float(r[m]);
      v[8 + m] = __uint_as_float(s[m]);
    }
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

// Eq. smat-state for one element given its keep decision, c and eps.
__device__ __forceinline__ float combine(bool kept, float c, float th, float t0, bool has_noise,
                                         float eps) {
  float x = t0;
  if (kept) x = (c == 1.0f) ? th : __fmaf_rn(c, __fsub_rn(th, t0), t0);
  if (has_noise) x = __fadd_rn(x, eps);
  return x;
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
template <int R, int DT, int NOISE, bool PE>
__global__ void __launch_bounds__(kBlock) simulate_kernel(const __grid_constant__ KArgs a) {
  for (int64_t ci = a.chunk_begin + blockIdx.x; ci < a.chunk_end; ci += gridDim.x) {
    const Chunk ch = a.chunks[ci];
    const DevTensor& T = a.tensors[ch.tensor];
    const TView v = make_view(T, a.scal[ch.tensor]);
    const void* th_p = T.theta;
    const void* t0_p = T.theta0;
    void* sim_p = T.sim;
    const bool vec = (v.flags & TF_VEC) != 0u;
    const bool masked = (v.flags & TF_MASK) != 0u;
    for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += 16 * (int64_t)kBlock) {
      const uint64_t g0 = (uint64_t)(v.off + i);
      if (vec && i + 16 <= ch.end) {
        float th[16], t0[16], out[16];
        load16<DT>(th_p, i, th);
        load16<DT>(t0_p, i, t0);
        const uint32_t keep = masked ? group_keep16<R>(a, v.tid, v.t_hi, v.t_lo, g0) : 0xFFFFu;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          float eps[4] = {0.0f, 0.0f, 0.0f, 0.0f};
          if (v.has_noise) noise4<NOISE>(stream_block<R>(a, S_NOISE, v.tid, (g0 >> 2) + q),
                                         v.noise_scale, eps);
          float c4[4] = {v.c, v.c, v.c, v.c};
          if (PE) {
            const uint4 w = stream_block<R>(a, S_ALPHA_E, v.tid, (g0 >> 2) + q);
            c4[0] = __fmul_rn(alpha_elem(a, w.x), v.inv_keep);
            c4[1] = __fmul_rn(alpha_elem(a, w.y), v.inv_keep);
            c4[2] = __fmul_rn(alpha_elem(a, w.z), v.inv_keep);
            c4[3] = __fmul_rn(alpha_elem(a, w.w), v.inv_keep);
          }
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int e = 4 * q + k;
            out[e] = combine((keep >> e) & 1u, c4[k], th[e], t0[e], v.has_noise, eps[k]);
          }
        }
        store16<DT>(sim_p, i, out);
      } else {
        const int64_t e_end = (i + 16 < ch.end) ? i + 16 : ch.end;
        for (int64_t e = i; e < e_end; ++e) {
          const uint64_t g = (uint64_t)(v.off + e);
          const bool kept = masked ? elem_kept<R>(a, v.tid, v.t_hi, v.t_lo, g) : true;
          float c = v.c;
          if (PE) {
            const uint4 w = stream_block<R>(a, S_ALPHA_E, v.tid, g >> 2);
            c = __fmul_rn(alpha_elem(a, pick(w, (unsigned)(g & 3))), v.inv_keep);
          }
          float eps = 0.0f;
          if (v.has_noise)
            eps = noise1<NOISE>(stream_block<R>(a, S_NOISE, v.tid, g >> 2), (unsigned)(g & 3),
                                v.noise_scale);
          store1<DT>(sim_p, e, combine(kept, c, load1<DT>(th_p, e), load1<DT>(t0_p, e), v.has_noise, eps));
        }
      }
    }
  }
}

// ---------------------------------------------------------- a5: gradient map ---
template <int R, int GDT, bool PE, bool ACC>
__global__ void __launch_bounds__(kBlock) gradmap_kernel(const __grid_constant__ KArgs a) {
  for (int64_t ci = a.chunk_begin + blockIdx.x; ci < a.chunk_end; ci += gridDim.x) {
    const Chunk ch = a.chunks[ci];
    const DevTensor& T = a.tensors[ch.tensor];
    const GradPtr G = a.grads[ch.tensor];
    const TView v = make_view(T, a.scal[ch.tensor]);
    const bool masked = (v.flags & TF_MASK) != 0u;
    for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += 16 * (int64_t)kBlock) {
      const uint64_t g0 = (uint64_t)(v.off + i);
      if (G.vec && i + 16 <= ch.end) {
        float gs[16], go[16], out[16];
        load16<GDT>(G.g_sim, i, gs);
        if (ACC) load16<GDT>(G.g_out, i, go);
        const uint32_t keep = masked ? group_keep16<R>(a, v.tid, v.t_hi, v.t_lo, g0) : 0xFFFFu;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          float c4[4] = {v.c, v.c, v.c, v.c};
          if (PE) {
            const uint4 w = stream_block<R>(a, S_ALPHA_E, v.tid, (g0 >> 2) + q);
            c4[0] = __fmul_rn(alpha_elem(a, w.x), v.inv_keep);
            c4[1] = __fmul_rn(alpha_elem(a, w.y), v.inv_keep);
            c4[2] = __fmul_rn(alpha_elem(a, w.z), v.inv_keep);
            c4[3] = __fmul_rn(alpha_elem(a, w.w), v.inv_keep);
          }
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int e = 4 * q + k;
            float g = ((keep >> e) & 1u) ? __fmul_rn(c4[k], gs[e]) : 0.0f;
            if (ACC) g = __fadd_rn(go[e], g);
            out[e] = g;
          }
        }
        store16<GDT>(G.g_out, i, out);
      } else {
        const int64_t e_end = (i + 16 < ch.end) ? i + 16 : ch.end;
        for (int64_t e = i; e < e_end; ++e) {
          const uint64_t g = (uint64_t)(v.off + e);
          const bool kept = masked ? elem_kept<R>(a, v.tid, v.t_hi, v.t_lo, g) : true;
          float c = v.c;
          if (PE) {
            const uint4 w = stream_block<R>(a, S_ALPHA_E, v.tid, g >> 2);
            c = __fmul_rn(alpha_elem(a, pick(w, (unsigned)(g & 3))), v.inv_keep);
          }
          float r = kept ? __fmul_rn(c, load1<GDT>(G.g_sim, e)) : 0.0f;
          if (ACC) r = __fadd_rn(load1<GDT>(G.g_out, e), r);
          store1<GDT>(G.g_out, e, r);
        }
      }
    }
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
        float th[16], t0[16];
        load16<DT>(T.theta, i, th);
        load16<DT>(T.theta0, i, t0);
#pragma unroll
        for (int k = 0; k < 16; ++k) {
          const float d = __fsub_rn(th[k], t0[k]);
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
    S.noise_scale = (NOISE == NOISE_UNIFORM) ? (float)(sqrt(3.0) * (double)sigma) : sigma;
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
      bits = group_keep16<R>(a, T.tid, T.t_hi, T.t_lo, g0) |
             (group_keep16<R>(a, T.tid, T.t_hi, T.t_lo, g0 + 16) << 16);
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
