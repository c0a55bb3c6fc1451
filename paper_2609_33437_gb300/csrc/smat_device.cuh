#pragma once
// SMAT simulated-merge device code for GB300 (sm_103a): shared helpers.
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
// All of them are multi-tensor launches over a chunk table (chunks of one
// tensor, 2^12 to 2^18 elements, the size chosen per list). The forward, with
// the statistics fused for sigma_rel tensors, is a persistent launch whose
// CTAs take whole chunks from an ordered work list; the unfused statistics,
// the grid-stride forward and the gradient map walk the table in grid-stride
// order. Each thread owns 16 consecutive elements at a time (one 256-bit load
// per bf16 input, two per fp32 input), which is exactly one Philox block of
// the mask stream (16 high bytes) and three blocks of the noise stream (24
// bits per element); with the 16-bit draw option, two blocks of each. The
// random words stay in registers; masks and noise are never written to
// memory.
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
constexpr int NOISE_LAPLACE = 2;
constexpr int NOISE_NONE = 3;  // sigma_t == 0: no add at all (chunk-level choice)

// Noise scale of each law at RMS sigma: uniform on [-sqrt3 sigma, sqrt3
// sigma], Gaussian sqrt2 sigma erfinv(v), Laplace (sigma / sqrt2) z(v).
template <int NOISE>
__device__ __forceinline__ float noise_scale_of(float sigma) {
  return (float)(sqrt(NOISE == NOISE_UNIFORM ? 3.0 : NOISE == NOISE_GAUSSIAN ? 2.0 : 0.5) * (double)sigma);
}
constexpr int DT_F32 = 0;
constexpr int DT_BF16 = 1;

// Stream variants. The `int R` template parameter of every kernel and helper
// that draws from the streams is a stream variant: the Philox rounds in its
// low byte (10, or 7 for the reduced-round option) and kDraw16 set for the
// 16-bit draw option, in which every per-element draw (Mask, Perturb,
// per-element Scale) is one 16-bit half of a Philox word: element gidx takes
// half gidx & 1 (low half first) of word (gidx & 7) >> 1 of block gidx >> 3,
// eight elements per block; the keep test is draw < floor(p_keep 2^16), with
// no low-bits part, and the noise draw u maps to (2u + 1 - 2^16) 2^-16.
template <int R>
constexpr bool draws16() { return (R & kDraw16) != 0; }  // kDraw16: smat_internal.h

// One Philox-4x32 block (the variant's rounds) with round keys precomputed
// from the seed. Each round takes the full 64-bit products of words 0 and 2
// with the round multipliers (one wide multiply each).
template <int R>
__device__ __forceinline__ uint4 philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                        const RoundKeys& k) {
  constexpr int kRounds = R & 0xFF;
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
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
__device__ __forceinline__ uint4 stream_block_at(const RoundKeys& key, uint32_t step, uint32_t stream,
                                                 uint32_t tid, uint64_t j) {
  return philox<R>((uint32_t)j, J0 ? 0u : (uint32_t)(j >> 32), (stream << 28) | tid, step, key);
}
template <int R, bool J0 = false>
__device__ __forceinline__ uint4 stream_block(const KArgs& a, uint32_t stream, uint32_t tid,
                                              uint64_t j) {
  return stream_block_at<R, J0>(a.key, a.step, stream, tid, j);
}

__device__ __forceinline__ uint32_t pick(const uint4& w, unsigned i) {
  return i == 0 ? w.x : (i == 1 ? w.y : (i == 2 ? w.z : w.w));
}

// u01(u) = (u >> 8) 2^-24 and sym24(u) = (2u + 1 - 2^24) 2^-24 (u a 24-bit
// field), both exact in fp32.
__device__ __forceinline__ float u01(uint32_t u) {
  return __fmul_rn(__uint2float_rn(u >> 8), 5.9604644775390625e-08f);
}
// sym24 as one conversion and one fused multiply-add: u 2^-23 and
// (2u + 1 - 2^24) 2^-24 = u 2^-23 - (1 - 2^-24) are exact in fp32 (|.| < 1,
// a multiple of 2^-24), so the single rounding of the FMA changes nothing.
constexpr float kSymScale = 1.1920928955078125e-07f;  // 2^-23
constexpr float kSymShift = -0.999999940395355224609375f;  // -(1 - 2^-24)
__device__ __forceinline__ float sym24(uint32_t u) {
  return __fmaf_rn(__uint2float_rn(u), kSymScale, kSymShift);
}

// erfinv(x) for |x| <= 1 - 2^-24 (every value sym24() produces), after the
// structure of M. Giles, "Approximating the erfinv function" (GPU Computing
// Gems Jade Edition, 2011), with coefficients fitted for this form by
// csrc/fit_erfinv.py: with L = log2(1 - x^2) (one fused multiply-add and the
// hardware log2),
//   L >= -8:  erfinv(x) = x * P(L)                 (degree 9, 99.8% of inputs)
//   L <  -8:  erfinv(x) = x * Q(sqrt(-L) - 3.8125)  (degree 9)
// Both ratios erfinv(x) / x are even in x, so the result is exactly odd.
// Relative error about 2e-7 (a few fp32 ulps); the tests bound it.
__device__ __forceinline__ float erfinv_poly(float x) {
  const float t = __fmaf_rn(-x, x, 1.0f);
  float L;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(L) : "f"(t));
  float p;
  if (L >= -8.0f) {
    p = 2.676246447e-10f;
    p = __fmaf_rn(p, L, 9.962457526e-09f);
    p = __fmaf_rn(p, L, 1.280022701e-07f);
    p = __fmaf_rn(p, L, 2.725655577e-07f);
    p = __fmaf_rn(p, L, -7.822631233e-06f);
    p = __fmaf_rn(p, L, -3.107573502e-05f);
    p = __fmaf_rn(p, L, 7.751958910e-04f);
    p = __fmaf_rn(p, L, 5.547157954e-03f);
    p = __fmaf_rn(p, L, -1.608200818e-01f);
    p = __fmaf_rn(p, L, 8.862268925e-01f);
  } else {
    const float v = __fsub_rn(sqrtf(-L), 3.8125f);
    p = 2.205743658e-05f;
    p = __fmaf_rn(p, v, -2.623226646e-05f);
    p = __fmaf_rn(p, v, -9.935771232e-05f);
    p = __fmaf_rn(p, v, 3.947049263e-04f);
    p = __fmaf_rn(p, v, -8.652319084e-04f);
    p = __fmaf_rn(p, v, 1.542331069e-03f);
    p = __fmaf_rn(p, v, -2.662600018e-03f);
    p = __fmaf_rn(p, v, 4.380439408e-03f);
    p = __fmaf_rn(p, v, 8.361965418e-01f);
    p = __fmaf_rn(p, v, 3.007633686e+00f);
  }
  return __fmul_rn(x, p);
}

// Packed fp32 pairs (sm_100 and later): two independent IEEE operations with
// round-to-nearest in one instruction. Written as PTX with an explicit .rn
// modifier: an operation with an explicit rounding mode is never contracted
// with a neighbour into a fused multiply-add, so each one rounds exactly as
// the specification's scalar operation does.
__device__ __forceinline__ float2 splat(float v) { return make_float2(v, v); }

__device__ __forceinline__ float2 mul2_rn(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "mul.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

__device__ __forceinline__ float2 add2_rn(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

__device__ __forceinline__ float2 sub2_rn(float2 a, float2 b) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "sub.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

__device__ __forceinline__ float2 fma2_rn(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}

// sym24 of two 24-bit noise fields: (2u + 1 - 2^24) 2^-24, exact. Two
// equivalent forms (identical values): an integer multiply-add, conversion
// and multiply, or a conversion and one fused multiply-add (see sym24). The
// Gaussian path measures faster with the second, the uniform path with the
// first.
template <bool FMA_FORM>
__device__ __forceinline__ float2 sym2(uint32_t u0, uint32_t u1) {
  if (FMA_FORM)
    return fma2_rn(make_float2(__uint2float_rn(u0), __uint2float_rn(u1)), splat(kSymScale), splat(kSymShift));
  const float2 m = make_float2(__int2float_rn(2 * (int)u0 + 1 - (1 << 24)), __int2float_rn(2 * (int)u1 + 1 - (1 << 24)));
  return mul2_rn(m, splat(5.9604644775390625e-08f));
}

// 16-bit option: (2u + 1 - 2^16) 2^-16 of two 16-bit draws as one conversion
// and one fused multiply-add, u 2^-15 - (1 - 2^-16): u 2^-15 is exact and so
// is the sum (a multiple of 2^-16 below 1 in magnitude).
constexpr float kSym16Scale = 3.0517578125e-05f;     // 2^-15
constexpr float kSym16Shift = -0.9999847412109375f;  // -(1 - 2^-16)
__device__ __forceinline__ float2 sym2_16(uint32_t u0, uint32_t u1) {
  return fma2_rn(make_float2(__uint2float_rn(u0), __uint2float_rn(u1)), splat(kSym16Scale), splat(kSym16Shift));
}
__device__ __forceinline__ float sym16(uint32_t u) {
  return __fmaf_rn(__uint2float_rn(u), kSym16Scale, kSym16Shift);
}
// The symmetric uniform of two draws of the variant (sym24 or sym16).
template <bool D16, bool FMA_FORM>
__device__ __forceinline__ float2 sym2v(uint32_t u0, uint32_t u1) {
  if constexpr (D16) return sym2_16(u0, u1);
  else return sym2<FMA_FORM>(u0, u1);
}

// The four 24-bit noise fields of a quad from its three noise words A, B, C:
// the top 24 bits of each word, and the three low bytes combined.
__device__ __forceinline__ void quad_fields(uint32_t A, uint32_t B, uint32_t C, uint32_t (&u)[4]) {
  u[0] = A >> 8;
  u[1] = B >> 8;
  u[2] = C >> 8;
  // bytes [x, A0, B0, C0] then drop x
  u[3] = __byte_perm(__byte_perm(A, B, 0x0400u), C, 0x4210u) >> 8;
}

// 16-bit option: the four draws of quad q (elements 4q .. 4q + 3) of a group,
// from the group's block q / 2 (its elements 8 (q / 2) .. 8 (q / 2) + 7):
// words 2 (q & 1) and 2 (q & 1) + 1, low half first (`hi` = q & 1).
__device__ __forceinline__ void halves_of(const uint4& b, int hi, uint32_t (&u)[4]) {
  const uint32_t w0 = hi ? b.z : b.x, w1 = hi ? b.w : b.y;
  u[0] = w0 & 0xFFFFu;
  u[1] = w0 >> 16;
  u[2] = w1 & 0xFFFFu;
  u[3] = w1 >> 16;
}

__device__ __forceinline__ float lg2_approx(float t) {
  float L;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(L) : "f"(t));
  return L;
}

// erfinv_poly on a pair: the central polynomial with packed multiply-adds
// when both lanes are central (99.6% of pairs), else lane by lane.
__device__ __forceinline__ float2 erfinv_poly2(float2 x) {
  const float2 t = fma2_rn(make_float2(-x.x, -x.y), x, splat(1.0f));
  const float2 L = make_float2(lg2_approx(t.x), lg2_approx(t.y));
  float2 p;
  if (fminf(L.x, L.y) >= -8.0f) {
    p = splat(2.676246447e-10f);
    p = fma2_rn(p, L, splat(9.962457526e-09f));
    p = fma2_rn(p, L, splat(1.280022701e-07f));
    p = fma2_rn(p, L, splat(2.725655577e-07f));
    p = fma2_rn(p, L, splat(-7.822631233e-06f));
    p = fma2_rn(p, L, splat(-3.107573502e-05f));
    p = fma2_rn(p, L, splat(7.751958910e-04f));
    p = fma2_rn(p, L, splat(5.547157954e-03f));
    p = fma2_rn(p, L, splat(-1.608200818e-01f));
    p = fma2_rn(p, L, splat(8.862268925e-01f));
    return mul2_rn(x, p);
  }
  return make_float2(erfinv_poly(x.x), erfinv_poly(x.y));
}

// Laplace(0, 1) variate of v in (-1, 1) by the inverse CDF, -sign(v) ln(1 -
// |v|): 1 - |v| is exact in fp32 for every noise-grid v, and log1pf of -|v|
// keeps full relative accuracy for small |v|.
__device__ __forceinline__ float laplace_unit(float v) {
  return copysignf(-log1pf(-fabsf(v)), v);
}

// The group path's erfinv of a pair: the central polynomial only (packed,
// branch free). minL collects the smallest L = log2(1 - x^2) seen, computed
// exactly as erfinv_poly computes it; an element with L < -8 belongs to the
// tail and its value here is wrong: the caller queues its group and rewrites
// it through the element path (erfinv_poly).
__device__ __forceinline__ float2 erfinv_central2(float2 x, float& minL) {
  const float2 t = fma2_rn(make_float2(-x.x, -x.y), x, splat(1.0f));
  const float2 L = make_float2(lg2_approx(t.x), lg2_approx(t.y));
  minL = fminf(minL, fminf(L.x, L.y));
  float2 p = splat(2.676246447e-10f);
  p = fma2_rn(p, L, splat(9.962457526e-09f));
  p = fma2_rn(p, L, splat(1.280022701e-07f));
  p = fma2_rn(p, L, splat(2.725655577e-07f));
  p = fma2_rn(p, L, splat(-7.822631233e-06f));
  p = fma2_rn(p, L, splat(-3.107573502e-05f));
  p = fma2_rn(p, L, splat(7.751958910e-04f));
  p = fma2_rn(p, L, splat(5.547157954e-03f));
  p = fma2_rn(p, L, splat(-1.608200818e-01f));
  p = fma2_rn(p, L, splat(8.862268925e-01f));
  return mul2_rn(x, p);
}

// Group-path noise of a pair (see erfinv_central2 for minL); D16: the two
// draws are 16-bit.
template <int NOISE, bool D16 = false>
__device__ __forceinline__ float2 noise_group2(uint32_t n0, uint32_t n1, float2 scale, float& minL) {
  if (NOISE == NOISE_UNIFORM) return mul2_rn(scale, sym2v<D16, false>(n0, n1));
  if (NOISE == NOISE_GAUSSIAN) return mul2_rn(scale, erfinv_central2(sym2v<D16, true>(n0, n1), minL));
  if (NOISE == NOISE_LAPLACE) {
    const float2 v = sym2v<D16, true>(n0, n1);
    return mul2_rn(scale, make_float2(laplace_unit(v.x), laplace_unit(v.y)));
  }
  return splat(0.0f);
}

// Perturb of one element from its 24-bit noise field u: uniform
// scale * sym24(u) with scale = fl(sqrt3 sigma), or Gaussian
// scale * erfinv(sym24(u)) with
// scale = fl(sqrt2 sigma) (inverse-CDF transform: sqrt2 erfinv(v) is
// N(0, 1) for v uniform on (-1, 1)).
template <int NOISE, bool D16 = false>
__device__ __forceinline__ float2 noise_of2(uint32_t n0, uint32_t n1, float2 scale) {
  if (NOISE == NOISE_UNIFORM) return mul2_rn(scale, sym2v<D16, false>(n0, n1));
  if (NOISE == NOISE_GAUSSIAN) return mul2_rn(scale, erfinv_poly2(sym2v<D16, true>(n0, n1)));
  if (NOISE == NOISE_LAPLACE) {
    const float2 v = sym2v<D16, true>(n0, n1);
    return mul2_rn(scale, make_float2(laplace_unit(v.x), laplace_unit(v.y)));
  }
  return splat(0.0f);
}

template <int NOISE, bool D16 = false>
__device__ __forceinline__ float noise_of(uint32_t u, float scale) {
  const float v = D16 ? sym16(u) : sym24(u);
  if (NOISE == NOISE_UNIFORM) return __fmul_rn(scale, v);
  if (NOISE == NOISE_GAUSSIAN) return __fmul_rn(scale, erfinv_poly(v));
  if (NOISE == NOISE_LAPLACE) return __fmul_rn(scale, laplace_unit(v));
  return 0.0f;
}

// The draw of one element (any alignment) in the NOISE or ALPHA_E stream: its
// packed 24-bit field, whose quad's three words come from one or two of the
// group's three blocks; or, with 16-bit draws, its half word.
template <int R>
__device__ __forceinline__ uint32_t field1(const KArgs& a, uint32_t stream, uint32_t tid, uint64_t gidx) {
  if constexpr (draws16<R>()) {
    const uint32_t w = pick(stream_block<R>(a, stream, tid, gidx >> 3), (unsigned)((gidx & 7) >> 1));
    return (gidx & 1) ? (w >> 16) : (w & 0xFFFFu);
  }
  const unsigned k = (unsigned)(gidx & 15), q = k >> 2, r = k & 3;
  const uint64_t j0 = 3 * (gidx >> 4);
  const unsigned s0 = 3 * q;  // first of the quad's words among the group's 12
  const uint4 lo = stream_block<R>(a, stream, tid, j0 + s0 / 4);
  const uint4 hi = (s0 / 4 == (s0 + 2) / 4) ? lo : stream_block<R>(a, stream, tid, j0 + (s0 + 2) / 4);
  const uint32_t w8[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
  // words s0, s0 + 1, s0 + 2 relative to block s0 / 4
  const unsigned b = s0 % 4;
  uint32_t ABC[3];
#pragma unroll
  for (int m = 0; m < 3; ++m) {
    const unsigned idx = b + m;  // 0..5; indices >= 4 fall in `hi`
    ABC[m] = idx == 0 ? w8[0] : idx == 1 ? w8[1] : idx == 2 ? w8[2] : idx == 3 ? w8[3] : idx == 4 ? w8[4] : w8[5];
  }
  uint32_t u[4];
  quad_fields(ABC[0], ABC[1], ABC[2], u);
  return r == 0 ? u[0] : r == 1 ? u[1] : r == 2 ? u[2] : u[3];
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
// bytes). Bit 8b + 7 of kw[q] is element 4q + b's flag. Returns whether some
// byte equals the threshold's high byte (probability 1/256 per element): such
// a tie is decided by the low 24 bits of the uniform (MASK_LO stream), which
// the caller resolves (group_ties16 / resolve_group_ties); its flag is left
// clear here.
__device__ __forceinline__ bool keep_bytes16(const uint4& w, uint32_t t_hi, uint32_t (&kw)[4]) {
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
  return anytie != 0u;
}
// 16-bit option: keep flags of the 16 elements gidx0 .. gidx0 + 15 (gidx0 %
// 16 == 0) from the two MASK blocks gidx0 / 8 and gidx0 / 8 + 1 (half h of
// word w serves element 2w + h), compared with T16 (< 2^16) two halves at a
// time (SWAR on 16-bit lanes, no borrow between them); the flags land in the
// byte layout of keep_bytes16 (bit 8b + 7 of kw[q] for element 4q + b).
__device__ __forceinline__ void keep_halves16(const uint4& b0, const uint4& b1, uint32_t t16, uint32_t (&kw)[4]) {
  const uint32_t words[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
  const uint32_t tt = t16 | (t16 << 16);
  const uint32_t tl = tt & 0x7FFF7FFFu;
  uint32_t f[8];
#pragma unroll
  for (int m = 0; m < 8; ++m) {
    const uint32_t x = words[m];
    // bit 15 of each half of d: low 15 bits of x >= low 15 bits of t
    const uint32_t d = (x | 0x80008000u) - tl;
    f[m] = ((~x & tt) | (~(x ^ tt) & ~d)) & 0x80008000u;  // x < t per half
  }
  // bytes 1 and 3 of words 2q and 2q + 1 carry elements 4q .. 4q + 3
#pragma unroll
  for (int q = 0; q < 4; ++q) kw[q] = __byte_perm(f[2 * q], f[2 * q + 1], 0x7531u);
}

// Keep flags of a group; true if some element's mask byte ties the
// threshold's (never with 16-bit draws, whose compare is exact).
template <int R, bool J0>
__device__ __forceinline__ bool group_keep16(const KArgs& a, uint32_t tid, uint32_t t_hi, uint64_t gidx0,
                                             uint32_t (&kw)[4]) {
  if constexpr (draws16<R>()) {
    keep_halves16(stream_block<R, J0>(a, S_MASK, tid, gidx0 >> 3), stream_block<R, J0>(a, S_MASK, tid, (gidx0 >> 3) + 1),
                  t_hi, kw);
    return false;
  }
  return keep_bytes16(stream_block<R, J0>(a, S_MASK, tid, gidx0 >> 4), t_hi, kw);
}

// Tie elements of the 16-element group at gidx0: bit e set iff element e's
// mask byte equals the threshold's high byte.
__device__ __forceinline__ uint32_t tie_bits16(const uint4& w, uint32_t t_hi) {
  const uint32_t words[4] = {w.x, w.y, w.z, w.w};
  const uint32_t tt = t_hi * 0x01010101u;
  uint32_t tbits = 0u;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint32_t e = words[q] ^ tt;
    const uint32_t eq = ~(((e & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | e) & 0x80808080u;  // exact per byte
    // bits 7, 15, 23, 31 -> bits 4q .. 4q + 3
    tbits |= ((((eq >> 7) * 0x00204081u) >> 21) & 0xFu) << (4 * q);
  }
  return tbits;
}
template <int R, bool J0>
__device__ __forceinline__ uint32_t group_ties16(const KArgs& a, uint32_t tid, uint32_t t_hi, uint64_t gidx0) {
  return tie_bits16(stream_block<R, J0>(a, S_MASK, tid, gidx0 >> 4), t_hi);
}

// Low-24-bit test of one tie element.
template <int R, bool J0>
__device__ __forceinline__ bool tie_kept(const KArgs& a, uint32_t tid, uint32_t t_lo, uint64_t gidx) {
  const uint4 l = stream_block<R, J0>(a, S_MASK_LO, tid, gidx >> 2);
  return (pick(l, (unsigned)(gidx & 3)) >> 8) < t_lo;
}

// Decide the ties of the group whose MASK block is w now (set their flags in kw).
template <int R, bool J0>
__device__ __forceinline__ void resolve_block_ties(const KArgs& a, uint32_t tid, uint32_t t_hi, uint32_t t_lo,
                                                   const uint4& w, uint64_t gidx0, uint32_t (&kw)[4]) {
  uint32_t tb = tie_bits16(w, t_hi);
  while (tb) {
    const int e = __ffs(tb) - 1;
    tb &= tb - 1u;
    if (tie_kept<R, J0>(a, tid, t_lo, gidx0 + (uint64_t)e)) set_kept(kw, e);
  }
}

// Set the flags of every tie element of the group whose MASK block is w.
__device__ __forceinline__ void set_tie_flags(const uint4& w, uint32_t t_hi, uint32_t (&kw)[4]) {
  const uint32_t words[4] = {w.x, w.y, w.z, w.w};
  const uint32_t tt = t_hi * 0x01010101u;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const uint32_t e = words[q] ^ tt;
    kw[q] |= ~(((e & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | e) & 0x80808080u;  // exact per byte
  }
}

// Whether a tie element is kept with probability at least 1/2 (t_lo / 2^24).
__device__ __forceinline__ bool tie_mostly_kept(uint32_t t_lo) { return t_lo >= (1u << 23); }

// Decide the group's ties now (set their flags in kw).
template <int R, bool J0>
__device__ __forceinline__ void resolve_group_ties(const KArgs& a, uint32_t tid, uint32_t t_hi, uint32_t t_lo,
                                                   uint64_t gidx0, uint32_t (&kw)[4]) {
  uint32_t tb = group_ties16<R, J0>(a, tid, t_hi, gidx0);
  while (tb) {
    const int e = __ffs(tb) - 1;
    tb &= tb - 1u;
    if (tie_kept<R, J0>(a, tid, t_lo, gidx0 + (uint64_t)e)) set_kept(kw, e);
  }
}

// Groups with tie elements whose low 24 mask bits are drawn at the end of the
// chunk, so the rare Philox calls run for the whole warp at once instead of
// once per group. Up to four 16-bit group indices per thread (a chunk has
// 4096 groups), two per register.
struct TieList {
  uint32_t w0 = 0u, w1 = 0u;
  int n = 0;
  __device__ __forceinline__ bool push(uint32_t g) {
    switch (n) {
      case 0: w0 = g; break;
      case 1: w0 |= g << 16; break;
      case 2: w1 = g; break;
      case 3: w1 |= g << 16; break;
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

// Keep decision of one element (any alignment) of the Mask stream at `step`.
template <int R>
__device__ __forceinline__ bool elem_kept_at(const RoundKeys& key, uint32_t step, uint32_t tid, uint32_t t_hi,
                                             uint32_t t_lo, uint64_t gidx) {
  if constexpr (draws16<R>()) {  // t_hi holds T16
    const uint32_t w = pick(stream_block_at<R>(key, step, S_MASK, tid, gidx >> 3), (unsigned)((gidx & 7) >> 1));
    return ((gidx & 1) ? (w >> 16) : (w & 0xFFFFu)) < t_hi;
  }
  const uint4 w = stream_block_at<R>(key, step, S_MASK, tid, gidx >> 4);
  const uint32_t hi = (pick(w, (unsigned)((gidx >> 2) & 3)) >> (8u * (unsigned)(gidx & 3))) & 0xFFu;
  if (hi != t_hi) return hi < t_hi;
  if (t_lo == 0u) return false;
  const uint4 l = stream_block_at<R>(key, step, S_MASK_LO, tid, gidx >> 2);
  return (pick(l, (unsigned)(gidx & 3)) >> 8) < t_lo;
}
template <int R>
__device__ __forceinline__ bool elem_kept(const KArgs& a, uint32_t tid, uint32_t t_hi,
                                          uint32_t t_lo, uint64_t gidx) {
  return elem_kept_at<R>(a.key, a.step, tid, t_hi, t_lo, gidx);
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
  // elements 2m and 2m + 1
  __device__ __forceinline__ float2 pair(int m) const {
    if (DT == DT_BF16) return make_float2(__uint_as_float(r[m] << 16), __uint_as_float(r[m] & 0xFFFF0000u));
    return make_float2(__uint_as_float(r[2 * m]), __uint_as_float(r[2 * m + 1]));
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

// Scale from a raw 32-bit word (per tensor, global): its top 24 bits.
__device__ __forceinline__ float alpha_elem(const KArgs& a, uint32_t u) {
  return __fmaf_rn(a.alpha_width, u01(u), a.alpha_min);
}

// Scale per element from its packed 24-bit ALPHA_E field: u 2^-24 is exact.
__device__ __forceinline__ float alpha_of24(const KArgs& a, uint32_t u24) {
  return __fmaf_rn(a.alpha_width, __fmul_rn(__uint2float_rn(u24), 5.9604644775390625e-08f), a.alpha_min);
}
// The same from a 16-bit draw (16-bit option): u 2^-16 is exact.
__device__ __forceinline__ float alpha_of16(const KArgs& a, uint32_t u16) {
  return __fmaf_rn(a.alpha_width, __fmul_rn(__uint2float_rn(u16), 1.52587890625e-05f), a.alpha_min);
}
template <bool D16>
__device__ __forceinline__ float alpha_of(const KArgs& a, uint32_t u) {
  return D16 ? alpha_of16(a, u) : alpha_of24(a, u);
}

// Per-chunk view of one tensor's constants.
struct TView {
  int64_t off;
  uint32_t tid, flags, t_hi, t_lo;
  float inv_keep, c, noise_scale;
  bool has_noise;
};

// Flags published by one CTA and waited for by another (work-list launches):
// a release store after the data, an acquire load before reading it. Every
// such wait gives up after kWaitLimit polls of 256 ns (about a second).
constexpr uint32_t kWaitLimit = 1u << 22;

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Wait until *p == v; false (and bit 0 of *error set) once the limit is reached.
__device__ __forceinline__ bool wait_value(const uint32_t* p, uint32_t v, int32_t* error) {
  for (uint32_t n = 0;; ++n) {
    if (ld_acquire(p) == v) return true;
    if (n >= kWaitLimit) {
      atomicOr(error, 1);
      return false;
    }
    __nanosleep(256);
  }
}

__device__ __forceinline__ double warp_sum(double x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
  return x;
}

// Row a2 for one chunk: sums of delta = theta - theta0 (each one fp32
// subtraction) and delta^2 over the chunk. Each thread keeps two 16-element
// groups of loads in flight and accumulates on fp32 pairs; the partial sums
// are combined in double in a fixed order (result valid on thread 0). All
// threads must call it.
template <int DT>
__device__ __forceinline__ void delta_group(const Raw16<DT>& th, const Raw16<DT>& t0, float2& s2, float2& q2) {
#pragma unroll
  for (int m = 0; m < 8; ++m) {
    const float2 a = th.pair(m), b = t0.pair(m);
    const float2 d = sub2_rn(a, b);
    s2 = add2_rn(s2, d);
    q2 = fma2_rn(d, d, q2);
  }
}

template <int DT>
__device__ __forceinline__ void chunk_delta_sums(const DevTensor& T, const Chunk& ch, double* sh_s,
                                                 double* sh_q, double& sum, double& sumsq) {
  constexpr int64_t kStride = 16 * (int64_t)kBlock;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool vec = (T.flags & TF_VEC) != 0u;
  float2 s2 = splat(0.0f), q2 = splat(0.0f);
  float s = 0.0f, q = 0.0f;
  for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += 2 * kStride) {
    const int64_t i2 = i + kStride;
    if (vec && i2 + 16 <= ch.end) {
      Raw16<DT> th1, t01, th2, t02;
      load16<DT>(T.theta, i, th1);
      load16<DT>(T.theta0, i, t01);
      load16<DT>(T.theta, i2, th2);
      load16<DT>(T.theta0, i2, t02);
      delta_group<DT>(th1, t01, s2, q2);
      delta_group<DT>(th2, t02, s2, q2);
    } else {
      for (int half = 0; half < 2; ++half) {
        const int64_t b = half ? i2 : i;
        if (b >= ch.end) break;
        if (vec && b + 16 <= ch.end) {
          Raw16<DT> th1, t01;
          load16<DT>(T.theta, b, th1);
          load16<DT>(T.theta0, b, t01);
          delta_group<DT>(th1, t01, s2, q2);
        } else {
          const int64_t e_end = (b + 16 < ch.end) ? b + 16 : ch.end;
          for (int64_t e = b; e < e_end; ++e) {
            const float d = __fsub_rn(load1<DT>(T.theta, e), load1<DT>(T.theta0, e));
            s = __fadd_rn(s, d);
            q = __fmaf_rn(d, d, q);
          }
        }
      }
    }
  }
  const double ds = warp_sum((double)s2.x + (double)s2.y + (double)s);
  const double dq = warp_sum((double)q2.x + (double)q2.y + (double)q);
  if (lane == 0) {
    sh_s[warp] = ds;
    sh_q[warp] = dq;
  }
  __syncthreads();
  sum = 0.0;
  sumsq = 0.0;
  if (threadIdx.x == 0) {
    for (int w = 0; w < kBlock / 32; ++w) {
      sum += sh_s[w];
      sumsq += sh_q[w];
    }
  }
  __syncthreads();
}

// sigma_t from the summed chunk sums of a tensor (population std of delta).
__device__ __forceinline__ float sigma_from_sums(double s, double q, int64_t n, float sigma_rel) {
  if (n <= 0) return 0.0f;
  const double dn = (double)n;
  const double mean = s / dn;
  double var = q / dn - mean * mean;
  if (var < 0.0) var = 0.0;
  return (float)((double)sigma_rel * sqrt(var));
}

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

}  // namespace
}  // namespace smat
