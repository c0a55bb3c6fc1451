// SMAT simulated-merge transform: plain single-threaded CPU oracle.
//
// TEST INFRASTRUCTURE ONLY. This file is the correctness reference for the
// CUDA path. Only tests/, the smoke check and the bench's CPU-baseline leg
// may load it. It shares no source, header, table or helper with the CUDA
// library: the Philox block, the stream layout, the bf16 rounding and the
// transforms below are written out independently from their definitions.
//
// What it computes (paper: "SMAT: Simple and Efficient Merge-Aware Training"):
//   forward   theta~ = theta0 + alpha * m (.) (theta - theta0) + eps
//             Eq. smat-state (Sec. 4.1), Scale / Mask / Perturb (Sec. 4.1,
//             Eq. smat-mask for m, uniform eps on [-sqrt3 sigma, sqrt3 sigma]).
//   gradient  g = alpha * m (.) g~                  Eq. smat-gradient (Sec. 4.2)
//   the mask is regenerated for the gradient, never stored (App. D,
//   "Implementation details").
//   update    the stored gradient fed into one decoupled-weight-decay AdamW
//             step of theta and fp32 moments (Sec. 4.3: theta updated with
//             the mapped gradient once the storage is switched back).
//
// The paper does not say how the random draws are produced. The counter-based
// stream layout below is this project's specification; every reading of the
// paper it relies on is listed in the design notes (readings R1-R15).
//
// Stream specification (both sides implement it; nothing here is shared):
//   Philox-4x32-R block (Salmon et al., SC'11), R = 10 by default.
//   key     = (seed mod 2^32, seed div 2^32)
//   counter = (j mod 2^32, j div 2^32, (stream << 28) | tensor_id, step)
//   W(stream, tid, j)[w] = word w of that block.
//   streams: MASK = 0, NOISE = 1, ALPHA_E = 2, ALPHA_T = 3, MASK_LO = 4.
//   gidx    = elem_offset + i  (global element index of local element i)
//   u01(u)      = (u >> 8) * 2^-24          in [0, 1)
//   Mask uniform U(gidx) in [0, 2^32):
//     hi = byte (gidx & 3) of W(MASK, tid, gidx >> 4)[(gidx >> 2) & 3]
//     lo = W(MASK_LO, tid, gidx >> 2)[gidx & 3] >> 8
//     U  = hi * 2^24 + lo ;  kept  <=>  U < T,  T = floor(p_keep * 2^32)
//   Packed 24-bit field F(stream, tid, gidx) of element gidx, k = gidx & 15,
//   q = k >> 2, r = k & 3:
//     S[0..11] = the 12 words of W(stream, tid, 3 (gidx >> 4) + b), b = 0, 1, 2
//     (S[4b + w] = word w of block b); the quad q uses A = S[3q], B = S[3q+1],
//     C = S[3q+2]: F = A >> 8, B >> 8, C >> 8 for r = 0, 1, 2, and for r = 3
//     F = (A & 255) | (B & 255) << 8 | (C & 255) << 16 (three words serve four
//     elements).
//   Noise field u = F(NOISE, tid, gidx);
//     sym24(u) = (2u + 1 - 2^24) 2^-24
//     uniform   eps = fl(sqrt3 sigma) * sym24(u)
//     Gaussian  eps = fl(sqrt2 sigma) * fl(erfinv(sym24(u)))  (inverse-CDF transform:
//               sqrt2 erfinv(v) is N(0, 1) for v uniform on (-1, 1))
//     Laplace   eps = fl(sigma / sqrt2) * fl(-sign(v) ln(1 - |v|)), v = sym24(u)
//               (inverse-CDF transform: -sign(v) ln(1 - |v|) is Laplace(0, 1),
//               variance 2, for v uniform on (-1, 1); the scale sigma / sqrt2 gives
//               RMS sigma, the matched-RMS comparison of Sec. 4.1 "Perturb")
//   Alpha:  per tensor  alpha = fma(amax - amin, u01(W(ALPHA_T, t_a, 0)[0]), amin)
//           t_a = 0x0FFFFFFF (one alpha for all tensors) or the tensor id;
//           per element alpha = fma(amax - amin, F(ALPHA_E, tid, gidx) 2^-24, amin)
//
//   The 16-bit draw option (draw_bits = 16; the layout above is draw_bits = 32):
//   each per-element draw is the 16-bit value
//     D(stream, tid, gidx) = half (gidx & 1), low half first, of word
//                            (gidx & 7) >> 1 of W(stream, tid, gidx >> 3)
//   (eight elements per block, no packing): Mask U16 = D(MASK, tid, gidx),
//   kept <=> U16 < T16 = floor(p_keep * 2^16) (no MASK_LO part); noise
//   v = sym16(D(NOISE, tid, gidx)) = (2u + 1 - 2^16) 2^-16 in place of sym24 in
//   every law; per element alpha = fma(amax - amin, D(ALPHA_E, tid, gidx) 2^-16,
//   amin). The per-tensor alpha is unchanged.
//
// Merging (the evaluation side, Eq. merged-state): theta_merge = theta0 +
// sum_j alpha_j (.) m_j (.) Delta_j over K experts, Delta_j = theta_j - theta0
// (one fp32 subtraction), accumulated over j = 0 .. K-1 in that order:
//   WA    acc = fma(fl(1/K), Delta_j, acc)             (weight averaging, Sec. 3.1)
//   TA    acc = fma(gamma, Delta_j, acc)               (Task Arithmetic, Sec. 3.1)
//   DARE  acc = fma(c, Delta_j, acc) for kept j only,  c = fl(gamma * fl(1 / p_keep)),
//         p_keep = fl(1 - p_drop); expert j's keep decision is the Mask stream
//         above with step = j (same threshold rule, same Philox draws)
//   TIES  trim: keep Delta_j where key(|Delta_j|) >= the r-th largest key of the
//         tensor's expert j, r = ceil(retention n) (key = the bits of |x| as
//         uint32; ties at the threshold are kept); elect s = sign of the fp32
//         sum over j of the trimmed values; merged = the fp32 mean of the
//         trimmed values of sign s (0 if none), acc = fl(gamma * merged)
//   theta_merge = fl(theta0 + acc), rounded to the storage dtype.
//
// Build: g++ -O2 -ffp-contract=off -shared -fPIC (no fast-math: every float
// operation below is one IEEE binary32 operation, round to nearest even).

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <functional>
#include <vector>

namespace {

// ---------------------------------------------------------------- Philox ---
// Philox-4x32-R as defined by Salmon, Moraes, Dror and Shaw, "Parallel Random
// Numbers: As Easy as 1, 2, 3" (SC'11): each round multiplies words 0 and 2
// by the two round multipliers, keeps both halves of the 64-bit products and
// mixes the high halves with words 1 and 3 and the round key; the key is
// bumped by the two Weyl increments between rounds.
const uint32_t kMulA = 0xD2511F53u;   // multiplier applied to counter word 0
const uint32_t kMulB = 0xCD9E8D57u;   // multiplier applied to counter word 2
const uint32_t kWeylA = 0x9E3779B9u;  // key word 0 increment (golden ratio)
const uint32_t kWeylB = 0xBB67AE85u;  // key word 1 increment (sqrt(3) - 1)

void philox_block(const uint32_t ctr[4], uint32_t k0, uint32_t k1, int rounds,
                  uint32_t out[4]) {
  uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  for (int r = 0; r < rounds; ++r) {
    if (r > 0) {
      k0 += kWeylA;
      k1 += kWeylB;
    }
    const uint64_t prodA = (uint64_t)kMulA * (uint64_t)x0;
    const uint64_t prodB = (uint64_t)kMulB * (uint64_t)x2;
    const uint32_t hiA = (uint32_t)(prodA >> 32), loA = (uint32_t)prodA;
    const uint32_t hiB = (uint32_t)(prodB >> 32), loB = (uint32_t)prodB;
    const uint32_t n0 = hiB ^ x1 ^ k0;
    const uint32_t n1 = loB;
    const uint32_t n2 = hiA ^ x3 ^ k1;
    const uint32_t n3 = loA;
    x0 = n0; x1 = n1; x2 = n2; x3 = n3;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

enum { S_MASK = 0, S_NOISE = 1, S_ALPHA_E = 2, S_ALPHA_T = 3, S_MASK_LO = 4 };
const uint32_t kGlobalAlphaId = 0x0FFFFFFFu;

enum { ALPHA_GLOBAL = 0, ALPHA_PER_TENSOR = 1, ALPHA_PER_ELEMENT = 2 };
enum { NOISE_UNIFORM = 0, NOISE_GAUSSIAN = 1, NOISE_LAPLACE = 2 };
enum { DT_F32 = 0, DT_BF16 = 1 };

}  // namespace

extern "C" {

// Layout mirrored by the ctypes wrapper (oracle/__init__.py).
struct OrcConfig {
  uint64_t seed;
  uint32_t step;
  int32_t rounds;      // Philox rounds (10 by default)
  int32_t alpha_mode;  // ALPHA_GLOBAL / ALPHA_PER_TENSOR / ALPHA_PER_ELEMENT
  int32_t noise;       // NOISE_UNIFORM / NOISE_GAUSSIAN / NOISE_LAPLACE
  float alpha_min;
  float alpha_max;
  int32_t draw_bits;   // 32 (the packed layout; 0 reads as 32) or 16 (the 16-bit draw option)
};

// AdamW hyperparameters of the fused gradient map + optimizer step.
struct OrcAdamW {
  float lr;
  float beta1;
  float beta2;
  float eps;
  float weight_decay;
  int32_t step;  // t >= 1: the optimizer's own step count (bias corrections)
};

struct OrcTensor {
  uint32_t tensor_id;  // < 0x0FFFFFFF
  int32_t dtype;       // parameter storage dtype
  int64_t numel;
  int64_t elem_offset;
  float keep_prob;     // p_keep = 1 - p (paper's p is the drop probability)
  float sigma;         // Perturb RMS when sigma_rel == 0
  float sigma_rel;     // > 0: sigma_t = sigma_rel * std_pop(theta - theta0)
};

}  // extern "C"

namespace {

uint32_t stream_word(const OrcConfig& cfg, uint32_t stream, uint32_t tid,
                     uint64_t j, unsigned w) {
  uint32_t ctr[4] = {(uint32_t)(j & 0xFFFFFFFFu), (uint32_t)(j >> 32),
                     (stream << 28) | tid, cfg.step};
  uint32_t out[4];
  philox_block(ctr, (uint32_t)(cfg.seed & 0xFFFFFFFFu), (uint32_t)(cfg.seed >> 32),
               cfg.rounds, out);
  return out[w];
}

const float kTwoPow24Inv = 5.9604644775390625e-08f;  // 2^-24, exact
const float kTwoPow16Inv = 1.52587890625e-05f;       // 2^-16, exact

bool draws16(const OrcConfig& cfg) { return cfg.draw_bits == 16; }

// 16-bit draw of element gidx in a per-element stream (the 16-bit option):
// half gidx & 1 (low half first) of word (gidx & 7) >> 1 of block gidx >> 3.
uint32_t draw16(const OrcConfig& cfg, uint32_t stream, uint32_t tid, uint64_t gidx) {
  const uint32_t w = stream_word(cfg, stream, tid, gidx >> 3, (unsigned)((gidx & 7) >> 1));
  return (gidx & 1) ? (w >> 16) : (w & 0xFFFFu);
}

float u01(uint32_t u) { return (float)(u >> 8) * kTwoPow24Inv; }

// ------------------------------------------------------------- bf16 I/O ---
float bf16_bits_to_f32(uint16_t h) {
  uint32_t b = (uint32_t)h << 16;
  float f;
  std::memcpy(&f, &b, 4);
  return f;
}

// Round to nearest even; NaN stays NaN (quiet bit set); overflow rounds to inf.
uint16_t f32_to_bf16_bits(float f) {
  uint32_t b;
  std::memcpy(&b, &f, 4);
  if ((b & 0x7F800000u) == 0x7F800000u && (b & 0x007FFFFFu) != 0u)
    return (uint16_t)((b >> 16) | 0x0040u);
  const uint32_t lsb = (b >> 16) & 1u;
  b += 0x7FFFu + lsb;
  return (uint16_t)(b >> 16);
}

float load_elem(const void* p, int dtype, int64_t i) {
  if (dtype == DT_BF16) return bf16_bits_to_f32(((const uint16_t*)p)[i]);
  return ((const float*)p)[i];
}

void store_elem(void* p, int dtype, int64_t i, float v) {
  if (dtype == DT_BF16)
    ((uint16_t*)p)[i] = f32_to_bf16_bits(v);
  else
    ((float*)p)[i] = v;
}

uint32_t stored_bits(int dtype, float v) {
  if (dtype == DT_BF16) return f32_to_bf16_bits(v);
  uint32_t b;
  std::memcpy(&b, &v, 4);
  return b;
}

// ------------------------------------------------------ per-call scalars ---
struct Scalars {
  float alpha;        // per-tensor alpha (unused in per-element mode)
  float inv_keep;     // 1 / p_keep  (Eq. smat-mask: 1 / (1 - p))
  float c;            // alpha * inv_keep
  uint64_t T;         // keep threshold on the 32-bit mask uniform (16-bit option: on U16)
  float sigma;        // Perturb RMS for this call
  float noise_scale;  // fl(sqrt3 sigma) (uniform), fl(sqrt2 sigma) (Gaussian), fl(sigma / sqrt2) (Laplace)
};

// Population mean and centred second moment of delta = theta - theta0 (each
// delta one fp32 subtraction), two passes in double.
void delta_moments(const OrcTensor& t, const void* th, const void* t0,
                   double* mean_out, double* m2_out) {
  if (t.numel <= 0) { *mean_out = 0.0; *m2_out = 0.0; return; }
  double s = 0.0;
  for (int64_t i = 0; i < t.numel; ++i) {
    const float d = load_elem(th, t.dtype, i) - load_elem(t0, t.dtype, i);
    s += (double)d;
  }
  const double mean = s / (double)t.numel;
  double m2 = 0.0;
  for (int64_t i = 0; i < t.numel; ++i) {
    const float d = load_elem(th, t.dtype, i) - load_elem(t0, t.dtype, i);
    const double e = (double)d - mean;
    m2 += e * e;
  }
  *mean_out = mean;
  *m2_out = m2;
}

float sigma_for(const OrcTensor& t, const void* th, const void* t0) {
  if (!(t.sigma_rel > 0.0f)) return t.sigma;
  if (t.numel <= 0) return 0.0f;
  double mean, m2;
  delta_moments(t, th, t0, &mean, &m2);
  return (float)((double)t.sigma_rel * std::sqrt(m2 / (double)t.numel));
}

// Scale (Sec. 4.1): alpha ~ U[alpha_min, alpha_max); Mask (Eq. smat-mask):
// keep with probability p_keep, rescale kept entries by 1 / p_keep; Perturb:
// uniform on [-sqrt3 sigma, sqrt3 sigma] (Sec. 4.1) or N(0, sigma^2).
Scalars make_scalars(const OrcConfig& cfg, const OrcTensor& t, float sigma) {
  Scalars s;
  const float width = cfg.alpha_max - cfg.alpha_min;
  if (cfg.alpha_mode == ALPHA_PER_ELEMENT) {
    s.alpha = 0.0f;
  } else {
    const uint32_t ta = (cfg.alpha_mode == ALPHA_GLOBAL) ? kGlobalAlphaId : t.tensor_id;
    s.alpha = std::fma(width, u01(stream_word(cfg, S_ALPHA_T, ta, 0, 0)), cfg.alpha_min);
  }
  s.inv_keep = (t.keep_prob > 0.0f) ? (float)(1.0 / (double)t.keep_prob) : 0.0f;
  s.c = s.alpha * s.inv_keep;
  s.T = (uint64_t)std::floor((double)t.keep_prob * (draws16(cfg) ? 65536.0 : 4294967296.0));
  s.sigma = sigma;
  s.noise_scale = (float)(std::sqrt(cfg.noise == NOISE_UNIFORM ? 3.0 : cfg.noise == NOISE_GAUSSIAN ? 2.0 : 0.5) *
                          (double)sigma);
  return s;
}

// ------------------------------------------------------- element values ---
bool is_kept(const OrcConfig& cfg, const OrcTensor& t, const Scalars& s, uint64_t gidx) {
  if (draws16(cfg)) return (uint64_t)draw16(cfg, S_MASK, t.tensor_id, gidx) < s.T;
  const uint32_t hw = stream_word(cfg, S_MASK, t.tensor_id, gidx >> 4, (unsigned)((gidx >> 2) & 3));
  const uint32_t hi = (hw >> (8u * (unsigned)(gidx & 3))) & 0xFFu;
  const uint32_t lo = stream_word(cfg, S_MASK_LO, t.tensor_id, gidx >> 2, (unsigned)(gidx & 3)) >> 8;
  const uint64_t U = ((uint64_t)hi << 24) | (uint64_t)lo;
  return U < s.T;
}

// 24-bit field of element gidx in a packed stream: the 12 words of blocks
// 3 (gidx >> 4) .. 3 (gidx >> 4) + 2 serve the group's 16 elements, three words
// per quad of four elements (the top 24 bits of each word for the quad's first
// three elements, the three low bytes for the fourth).
uint32_t field24(const OrcConfig& cfg, uint32_t stream, uint32_t tid, uint64_t gidx) {
  const unsigned k = (unsigned)(gidx & 15), q = k >> 2, r = k & 3;
  uint32_t quad[3];
  for (unsigned m = 0; m < 3; ++m) {
    const unsigned s_idx = 3 * q + m;  // index into the 12 words of the 3 blocks
    quad[m] = stream_word(cfg, stream, tid, 3 * (gidx >> 4) + s_idx / 4, s_idx % 4);
  }
  if (r < 3) return quad[r] >> 8;
  return (quad[0] & 0xFFu) | ((quad[1] & 0xFFu) << 8) | ((quad[2] & 0xFFu) << 16);
}

// Scale per coordinate: alpha ~ U[alpha_min, alpha_max) from the element's
// 24-bit ALPHA_E field (16-bit option: its 16-bit draw), then c = alpha /
// p_keep (Eq. smat-mask rescale).
float element_c(const OrcConfig& cfg, const OrcTensor& t, const Scalars& s, uint64_t gidx) {
  if (cfg.alpha_mode != ALPHA_PER_ELEMENT) return s.c;
  const float width = cfg.alpha_max - cfg.alpha_min;
  const float u01e = draws16(cfg) ? (float)draw16(cfg, S_ALPHA_E, t.tensor_id, gidx) * kTwoPow16Inv
                                  : (float)field24(cfg, S_ALPHA_E, t.tensor_id, gidx) * kTwoPow24Inv;
  const float alpha = std::fma(width, u01e, cfg.alpha_min);
  return alpha * s.inv_keep;
}

// erfinv(v) for -1 < v < 1 in double: the root y of erf(y) = |v| (or, for
// |v| > 1/2, of erfc(y) = 1 - |v|, which is exact in double for the 24-bit
// values sym() produces), by safeguarded Newton steps from a bracket.
double erfinv_d(double v) {
  if (v == 0.0) return 0.0;
  const double a = std::fabs(v);
  const bool tail = a > 0.5;
  const double r = 1.0 - a;  // exact for a = odd multiple of 2^-24
  const double two_over_sqrt_pi = 1.1283791670955126;
  double lo = 0.0, hi = 6.0;  // erf(6) = 1 - 2e-17 exceeds every input
  double y = tail ? std::sqrt(-std::log(r * (2.0 - r))) : a * 0.886226925452758;
  if (!(y > lo && y < hi)) y = 0.5 * (lo + hi);
  for (int it = 0; it < 200; ++it) {
    // f(y) increasing in y: erf(y) - a, or (1 - a) - erfc(y) in the tail
    const double f = tail ? (r - std::erfc(y)) : (std::erf(y) - a);
    if (f > 0.0) hi = y; else lo = y;
    const double fp = two_over_sqrt_pi * std::exp(-y * y);
    double yn = y - f / fp;
    if (!(yn > lo && yn < hi)) yn = 0.5 * (lo + hi);
    if (std::fabs(yn - y) <= 1e-17 * y || hi - lo <= 1e-17 * y) { y = yn; break; }
    y = yn;
  }
  return v < 0.0 ? -y : y;
}

// 24-bit noise field of element gidx (three noise words serve four elements).
uint32_t noise_field(const OrcConfig& cfg, const OrcTensor& t, uint64_t gidx) {
  return field24(cfg, S_NOISE, t.tensor_id, gidx);
}

double sym24_d(uint32_t u24) { return (double)(2 * (int64_t)u24 + 1 - (1 << 24)) * 0x1p-24; }
double sym16_d(uint32_t u16) { return (double)(2 * (int64_t)u16 + 1 - (1 << 16)) * 0x1p-16; }

// The symmetric uniform v in (-1, 1) of element gidx's noise draw: sym24 of its
// 24-bit field, or sym16 of its 16-bit draw. Exact in fp32 and double (an odd
// multiple of 2^-24 or 2^-16 below 1 in magnitude).
double noise_v(const OrcConfig& cfg, const OrcTensor& t, uint64_t gidx) {
  if (draws16(cfg)) return sym16_d(draw16(cfg, S_NOISE, t.tensor_id, gidx));
  return sym24_d(noise_field(cfg, t, gidx));
}

// Laplace(0, 1) variate of v in (-1, 1) by the inverse CDF: -sign(v) ln(1 - |v|).
double laplace_d(double v) {
  const double z = -std::log1p(-std::fabs(v));
  return v < 0.0 ? -z : z;
}

// Unit-variance normal variate of element gidx: sqrt2 erfinv(v).
double gauss_z(const OrcConfig& cfg, const OrcTensor& t, uint64_t gidx) {
  return std::sqrt(2.0) * erfinv_d(noise_v(cfg, t, gidx));
}

float noise_eps(const OrcConfig& cfg, const OrcTensor& t, const Scalars& s, uint64_t gidx) {
  const double v = noise_v(cfg, t, gidx);
  if (cfg.noise == NOISE_UNIFORM) return s.noise_scale * (float)v;
  if (cfg.noise == NOISE_LAPLACE) return s.noise_scale * (float)laplace_d(v);
  return s.noise_scale * (float)erfinv_d(v);
}

// Eq. smat-state for one element, fp32 arithmetic, before the storage rounding.
float simulate_value(const OrcConfig& cfg, const OrcTensor& t, const Scalars& s,
                     uint64_t gidx, float th, float t0) {
  float x;
  if (is_kept(cfg, t, s, gidx)) {
    const float c = element_c(cfg, t, s, gidx);
    const float d = th - t0;
    x = (c == 1.0f) ? th : std::fma(c, d, t0);
  } else {
    x = t0;
  }
  if (s.sigma > 0.0f) x = x + noise_eps(cfg, t, s, gidx);
  return x;
}

// Eq. smat-gradient for one element, fp32, before the storage rounding.
float gradmap_value(const OrcConfig& cfg, const OrcTensor& t, const Scalars& s,
                    uint64_t gidx, float gsim, int accumulate, float gold) {
  float g = 0.0f;
  if (is_kept(cfg, t, s, gidx)) g = element_c(cfg, t, s, gidx) * gsim;
  if (accumulate) g = gold + g;
  return g;
}

}  // namespace

extern "C" {

// One Philox-4x32-R block.
void orc_philox(const uint32_t* ctr4, const uint32_t* key2, int32_t rounds, uint32_t* out4) {
  philox_block(ctr4, key2[0], key2[1], rounds, out4);
}

// Raw stream word W(stream, tid, j)[w] for n (j, w) pairs.
void orc_stream_words(const OrcConfig* cfg, uint32_t stream, uint32_t tid, const uint64_t* j,
                      const uint32_t* w, int64_t n, uint32_t* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = stream_word(*cfg, stream, tid, j[i], w[i] & 3u);
}

// fp32 <-> bf16 bit conversions (storage rounding of the oracle).
void orc_f32_to_bf16(const float* x, int64_t n, uint16_t* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = f32_to_bf16_bits(x[i]);
}

// erfinv in double (the Gaussian transform's definition), for its pin.
void orc_erfinv(const double* v, int64_t n, double* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = erfinv_d(v[i]);
}

// The Laplace transform -sign(v) ln(1 - |v|) in double, for its pins.
void orc_laplace(const double* v, int64_t n, double* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = laplace_d(v[i]);
}

// Unit-variance variate of each element's noise under the config's law:
// sqrt3 v (uniform), sqrt2 erfinv(v) (Gaussian), laplace(v) / sqrt2 (Laplace),
// v the element's symmetric uniform (noise_v).
void orc_noise_z(const OrcConfig* cfg, const OrcTensor* t, const uint64_t* gidx, int64_t n, double* z) {
  for (int64_t k = 0; k < n; ++k) {
    const double v = noise_v(*cfg, *t, gidx[k]);
    z[k] = cfg->noise == NOISE_UNIFORM    ? std::sqrt(3.0) * v
           : cfg->noise == NOISE_GAUSSIAN ? std::sqrt(2.0) * erfinv_d(v)
                                          : laplace_d(v) / std::sqrt(2.0);
  }
}

// Per-call scalars: out = {alpha, inv_keep, c, T, sigma_t, noise_scale}.
// theta / theta0 are read only when sigma_rel > 0.
void orc_scalars(const OrcConfig* cfg, const OrcTensor* t, const void* th, const void* t0,
                 double* out6) {
  const Scalars s = make_scalars(*cfg, *t, sigma_for(*t, th, t0));
  out6[0] = s.alpha; out6[1] = s.inv_keep; out6[2] = s.c;
  out6[3] = (double)s.T; out6[4] = s.sigma; out6[5] = s.noise_scale;
}

// delta statistics: out = {mean, M2, sigma_t}.
void orc_delta_stats(const OrcTensor* t, const void* th, const void* t0, double* out3) {
  double mean, m2;
  delta_moments(*t, th, t0, &mean, &m2);
  out3[0] = mean; out3[1] = m2; out3[2] = sigma_for(*t, th, t0);
}

// Forward over a whole tensor: out[i] = round_dtype(Eq. smat-state).
void orc_simulate(const OrcConfig* cfg, const OrcTensor* t, const void* th, const void* t0,
                  void* out) {
  const Scalars s = make_scalars(*cfg, *t, sigma_for(*t, th, t0));
  for (int64_t i = 0; i < t->numel; ++i) {
    const uint64_t gidx = (uint64_t)(t->elem_offset + i);
    const float v = simulate_value(*cfg, *t, s, gidx, load_elem(th, t->dtype, i),
                                   load_elem(t0, t->dtype, i));
    store_elem(out, t->dtype, i, v);
  }
}

// Forward at sampled local indices with a given sigma_t; th_vals / t0_vals are
// the fp32 values of theta / theta0 there. out_bits: stored bits (bf16 in the
// low 16 bits); kept_out: 1 if the element was kept.
void orc_simulate_at(const OrcConfig* cfg, const OrcTensor* t, float sigma_t, const int64_t* idx,
                     int64_t n, const float* th_vals, const float* t0_vals, uint32_t* out_bits,
                     uint8_t* kept_out) {
  const Scalars s = make_scalars(*cfg, *t, sigma_t);
  for (int64_t k = 0; k < n; ++k) {
    const uint64_t gidx = (uint64_t)(t->elem_offset + idx[k]);
    const float v = simulate_value(*cfg, *t, s, gidx, th_vals[k], t0_vals[k]);
    out_bits[k] = stored_bits(t->dtype, v);
    if (kept_out) kept_out[k] = is_kept(*cfg, *t, s, gidx) ? 1 : 0;
  }
}

// Gradient map over a whole tensor: g_out[i] = round_gdtype(Eq. smat-gradient
// [+ g_out[i] when accumulating]). g_out may equal g_sim when not accumulating.
void orc_gradmap(const OrcConfig* cfg, const OrcTensor* t, int32_t gdtype, int32_t accumulate,
                 const void* g_sim, void* g_out) {
  const Scalars s = make_scalars(*cfg, *t, 0.0f);
  for (int64_t i = 0; i < t->numel; ++i) {
    const uint64_t gidx = (uint64_t)(t->elem_offset + i);
    const float gold = accumulate ? load_elem(g_out, gdtype, i) : 0.0f;
    const float v = gradmap_value(*cfg, *t, s, gidx, load_elem(g_sim, gdtype, i), accumulate, gold);
    store_elem(g_out, gdtype, i, v);
  }
}

// Gradient map fused with the optimizer step of the simulated-loss step
// (Sec. 4.3: the mapped gradient updates the original storage theta), here
// AdamW with decoupled weight decay (Loshchilov and Hutter, ICLR 2019) and
// fp32 moments. Per element, one IEEE binary32 operation at a time:
//   g   = the value the gradient map stores (Eq. smat-gradient, rounded to the
//         gradient dtype), so the fused step equals the gradient map followed
//         by the update
//   th  = th * decay,                 decay = fl(1 - lr wd)
//   m1  = b1 m1 + omb1 g,             omb1  = fl(1 - b1)
//   m2  = b2 m2 + omb2 (g g),         omb2  = fl(1 - b2)
//   den = sqrt(m2) / bc2 + eps,       bc2   = fl(sqrt(1 - b2^t))
//   th  = th - step (m1 / den),       step  = fl(lr / (1 - b1^t))
// with the per-call constants computed in double and rounded once; theta is
// then rounded to its storage dtype. theta is updated in place (dtype of the
// tensor), m1 and m2 are fp32 arrays updated in place.
namespace {
struct AdamConsts {
  float decay, omb1, omb2, bc2, step;
};

AdamConsts adam_consts(const OrcAdamW& o) {
  const double b1 = o.beta1, b2 = o.beta2, tt = (double)o.step;
  AdamConsts k;
  k.decay = (float)(1.0 - (double)o.lr * (double)o.weight_decay);
  k.omb1 = (float)(1.0 - b1);
  k.omb2 = (float)(1.0 - b2);
  k.bc2 = (float)std::sqrt(1.0 - std::pow(b2, tt));
  k.step = (float)((double)o.lr / (1.0 - std::pow(b1, tt)));
  return k;
}

// One element: the stored gradient (Eq. smat-gradient, rounded to the
// gradient dtype and read back), then the update above; returns theta
// before its rounding to the storage dtype.
float adam_element(const OrcConfig& cfg, const OrcTensor& t, const Scalars& s, const OrcAdamW& o,
                   const AdamConsts& k, int32_t gdtype, uint64_t gidx, float g_sim, float th, float& m1,
                   float& m2) {
  float g = gradmap_value(cfg, t, s, gidx, g_sim, 0, 0.0f);
  if (gdtype == DT_BF16) g = bf16_bits_to_f32(f32_to_bf16_bits(g));
  th = th * k.decay;
  m1 = o.beta1 * m1 + k.omb1 * g;
  m2 = o.beta2 * m2 + k.omb2 * (g * g);
  const float den = std::sqrt(m2) / k.bc2 + o.eps;
  return th - k.step * (m1 / den);
}
}  // namespace

void orc_gradmap_adamw(const OrcConfig* cfg, const OrcTensor* t, int32_t gdtype, const void* g_sim,
                       void* theta, float* m1, float* m2, const OrcAdamW* o) {
  const Scalars s = make_scalars(*cfg, *t, 0.0f);
  const AdamConsts k = adam_consts(*o);
  for (int64_t i = 0; i < t->numel; ++i) {
    const float th = adam_element(*cfg, *t, s, *o, k, gdtype, (uint64_t)(t->elem_offset + i),
                                  load_elem(g_sim, gdtype, i), load_elem(theta, t->dtype, i), m1[i], m2[i]);
    store_elem(theta, t->dtype, i, th);
  }
}

// The same at sampled local indices: g~ and theta given as fp32 values, the
// moments updated in place, theta returned as its stored bits.
void orc_gradmap_adamw_at(const OrcConfig* cfg, const OrcTensor* t, int32_t gdtype, const int64_t* idx,
                          int64_t n, const float* gsim_vals, const float* theta_vals, float* m1, float* m2,
                          const OrcAdamW* o, uint32_t* theta_bits) {
  const Scalars s = make_scalars(*cfg, *t, 0.0f);
  const AdamConsts k = adam_consts(*o);
  for (int64_t j = 0; j < n; ++j) {
    const float th = adam_element(*cfg, *t, s, *o, k, gdtype, (uint64_t)(t->elem_offset + idx[j]), gsim_vals[j],
                                  theta_vals[j], m1[j], m2[j]);
    theta_bits[j] = stored_bits(t->dtype, th);
  }
}

// Gradient map at sampled local indices (values given in fp32).
void orc_gradmap_at(const OrcConfig* cfg, const OrcTensor* t, int32_t gdtype, int32_t accumulate,
                    const int64_t* idx, int64_t n, const float* gsim_vals, const float* gold_vals,
                    uint32_t* out_bits) {
  const Scalars s = make_scalars(*cfg, *t, 0.0f);
  for (int64_t k = 0; k < n; ++k) {
    const uint64_t gidx = (uint64_t)(t->elem_offset + idx[k]);
    const float gold = accumulate ? gold_vals[k] : 0.0f;
    out_bits[k] = stored_bits(gdtype, gradmap_value(*cfg, *t, s, gidx, gsim_vals[k], accumulate, gold));
  }
}

// Packed keep bits: bit (i mod 32) of word i / 32, LSB first; unused high bits of
// the last word are 0.
void orc_mask_bits(const OrcConfig* cfg, const OrcTensor* t, uint32_t* bits) {
  const Scalars s = make_scalars(*cfg, *t, 0.0f);
  const int64_t nwords = (t->numel + 31) / 32;
  for (int64_t w = 0; w < nwords; ++w) bits[w] = 0u;
  for (int64_t i = 0; i < t->numel; ++i) {
    const uint64_t gidx = (uint64_t)(t->elem_offset + i);
    if (is_kept(*cfg, *t, s, gidx)) bits[i >> 5] |= (1u << (i & 31));
  }
}

// Unit-variance normal variates z = sqrt2 erfinv(sym(n)) of the Gaussian mode.
void orc_gauss_z(const OrcConfig* cfg, const OrcTensor* t, const uint64_t* gidx, int64_t n,
                 double* z) {
  for (int64_t k = 0; k < n; ++k) z[k] = gauss_z(*cfg, *t, gidx[k]);
}

// Real-arithmetic (double) evaluation of the same transform, for the
// finite-difference check of Eq. smat-gradient. The draws and the per-call
// scalars are those of the fp32 path; the arithmetic is double.
void orc_simulate_f64(const OrcConfig* cfg, const OrcTensor* t, float sigma_t, const double* th,
                      const double* t0, double* out) {
  const Scalars s = make_scalars(*cfg, *t, sigma_t);
  for (int64_t i = 0; i < t->numel; ++i) {
    const uint64_t gidx = (uint64_t)(t->elem_offset + i);
    double x = t0[i];
    if (is_kept(*cfg, *t, s, gidx)) {
      const double c = (double)element_c(*cfg, *t, s, gidx);
      x = t0[i] + c * (th[i] - t0[i]);
    }
    if (s.sigma > 0.0f) {
      const double v = noise_v(*cfg, *t, gidx);
      if (cfg->noise == NOISE_UNIFORM)
        x += (double)s.noise_scale * v;
      else if (cfg->noise == NOISE_LAPLACE)
        x += (double)s.noise_scale * laplace_d(v);
      else
        x += (double)s.noise_scale * erfinv_d(v);
    }
    out[i] = x;
  }
}

void orc_gradmap_f64(const OrcConfig* cfg, const OrcTensor* t, const double* gsim, double* out) {
  const Scalars s = make_scalars(*cfg, *t, 0.0f);
  for (int64_t i = 0; i < t->numel; ++i) {
    const uint64_t gidx = (uint64_t)(t->elem_offset + i);
    out[i] = is_kept(*cfg, *t, s, gidx) ? (double)element_c(*cfg, *t, s, gidx) * gsim[i] : 0.0;
  }
}

}  // extern "C"

// ------------------------------------------------------------- merging ---
namespace {

enum { MERGE_WA = 0, MERGE_TA = 1, MERGE_DARE_TA = 2, MERGE_TIES = 3 };

}  // namespace

extern "C" {

// Layout mirrored by the ctypes wrapper (oracle/__init__.py).
struct OrcMerge {
  uint64_t seed;
  int32_t rounds;
  int32_t method;     // MERGE_*
  int32_t n_experts;  // K >= 1
  float gamma;        // merging coefficient (TA, DARE, TIES)
  float p_drop;       // DARE drop probability in [0, 1)
  float retention;    // TIES fraction kept per expert, (0, 1]
};

}  // extern "C"

namespace {

uint32_t abs_key(float x) {
  uint32_t b;
  std::memcpy(&b, &x, 4);
  return b & 0x7FFFFFFFu;
}

// The r-th largest key of one expert's task vector, r = ceil(retention n)
// clamped to [1, n] (sort in descending order and index: plain, not fast).
uint32_t orc_ties_threshold_of(const std::vector<float>& delta, double retention) {
  const int64_t n = (int64_t)delta.size();
  if (n == 0) return 0u;
  int64_t r = (int64_t)std::ceil(retention * (double)n);
  if (r < 1) r = 1;
  if (r > n) r = n;
  std::vector<uint32_t> keys((size_t)n);
  for (int64_t i = 0; i < n; ++i) keys[(size_t)i] = abs_key(delta[(size_t)i]);
  std::sort(keys.begin(), keys.end(), std::greater<uint32_t>());
  return keys[(size_t)(r - 1)];
}

}  // namespace

extern "C" {

// One tensor: theta0 and the K experts (dtype storage, n elements each) into
// out; thresholds_out (K entries, may be NULL) receives the TIES keys.
void orc_merge(const OrcMerge* m, uint32_t tensor_id, int32_t dtype, int64_t n, int64_t elem_offset,
               const void* theta0, const void* const* experts, void* out, uint32_t* thresholds_out) {
  const int K = m->n_experts;
  std::vector<std::vector<float>> delta((size_t)K, std::vector<float>((size_t)n));
  for (int e = 0; e < K; ++e)
    for (int64_t i = 0; i < n; ++i)
      delta[(size_t)e][(size_t)i] = load_elem(experts[e], dtype, i) - load_elem(theta0, dtype, i);
  std::vector<uint32_t> thr((size_t)K, 0u);
  if (m->method == MERGE_TIES)
    for (int e = 0; e < K; ++e) thr[(size_t)e] = orc_ties_threshold_of(delta[(size_t)e], (double)m->retention);
  if (thresholds_out)
    for (int e = 0; e < K; ++e) thresholds_out[e] = thr[(size_t)e];
  // DARE: the Mask stream of Eq. smat-mask at step = expert index
  const float keep = 1.0f - m->p_drop;
  OrcTensor mt;
  mt.tensor_id = tensor_id;
  mt.dtype = dtype;
  mt.numel = n;
  mt.elem_offset = elem_offset;
  mt.keep_prob = keep;
  mt.sigma = 0.0f;
  mt.sigma_rel = 0.0f;
  const float inv_keep = keep > 0.0f ? (float)(1.0 / (double)keep) : 0.0f;
  const float c_dare = m->gamma * inv_keep;
  const float c_wa = (float)(1.0 / (double)K);
  for (int64_t i = 0; i < n; ++i) {
    const uint64_t gidx = (uint64_t)(elem_offset + i);
    float acc = 0.0f;
    if (m->method == MERGE_TIES) {
      float sum = 0.0f;
      for (int e = 0; e < K; ++e) {
        const float d = delta[(size_t)e][(size_t)i];
        if (abs_key(d) >= thr[(size_t)e]) sum = sum + d;
      }
      const int s = sum > 0.0f ? 1 : (sum < 0.0f ? -1 : 0);
      float part = 0.0f;
      int cnt = 0;
      for (int e = 0; e < K; ++e) {
        const float d = delta[(size_t)e][(size_t)i];
        if (abs_key(d) < thr[(size_t)e]) continue;
        if ((s > 0 && d > 0.0f) || (s < 0 && d < 0.0f)) {
          part = part + d;
          ++cnt;
        }
      }
      const float merged = cnt > 0 ? part / (float)cnt : 0.0f;
      acc = m->gamma * merged;
    } else {
      for (int e = 0; e < K; ++e) {
        const float d = delta[(size_t)e][(size_t)i];
        if (m->method == MERGE_WA) {
          acc = std::fma(c_wa, d, acc);
        } else if (m->method == MERGE_TA) {
          acc = std::fma(m->gamma, d, acc);
        } else {
          OrcConfig cfg;
          cfg.seed = m->seed;
          cfg.step = (uint32_t)e;
          cfg.rounds = m->rounds;
          cfg.alpha_mode = ALPHA_PER_TENSOR;
          cfg.noise = NOISE_UNIFORM;
          cfg.alpha_min = 0.0f;
          cfg.alpha_max = 1.0f;
          cfg.draw_bits = 32;  // DARE masks use the packed mask layout
          Scalars s;
          s.T = (uint64_t)std::floor((double)keep * 4294967296.0);
          if (is_kept(cfg, mt, s, gidx)) acc = std::fma(c_dare, d, acc);
        }
      }
    }
    store_elem(out, dtype, i, load_elem(theta0, dtype, i) + acc);
  }
}

}  // extern "C"
