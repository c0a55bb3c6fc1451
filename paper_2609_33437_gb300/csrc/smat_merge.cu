// Merging over K experts (the evaluation side, Eq. merged-state):
// theta_merge = theta0 + sum_j alpha_j (.) m_j (.) Delta_j, Delta_j = theta_j -
// theta0, for weight averaging, Task Arithmetic, DARE followed by Task
// Arithmetic and TIES (the merging methods of Sec. 5). Elementwise and bound
// by HBM bandwidth: each element reads theta0 and the K experts once and
// writes the result once (TIES first reads every expert three more times to
// select its per-tensor trim thresholds exactly).
//
// Arithmetic, identical to the CPU oracle: Delta_j one fp32 subtraction;
// experts accumulated in index order, one fused multiply-add each (WA 1/K,
// TA gamma, DARE gamma / p_keep on the kept coordinates); TIES sums the kept
// values, elects the sign of that sum, averages the kept values of that sign
// (one fp32 division) and scales by gamma; then fl(theta0 + acc) rounded to
// the storage dtype. DARE's mask of expert j is the library's Mask stream
// with step = j.
//
// TIES trim threshold of each (tensor, expert): the r-th largest key of
// |Delta_j| (key = the bits of the magnitude as uint32, r = ceil(retention
// n)), found by a most-significant-digit radix select in three passes of 11,
// 11 and 10 bits: each pass histograms the digit of the keys that match the
// digits decided so far (shared-memory histograms per chunk, flushed into
// 64-bit global bins), then one CTA per (tensor, expert) picks the digit
// whose bin holds the r-th largest and the rank within it.

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <unordered_set>
#include <vector>

#include "smat.h"
#include "smat_device.cuh"

namespace smat {
namespace {

constexpr int kMergeMaxExperts = SMAT_MERGE_MAX_EXPERTS;
constexpr int64_t kMergeChunk = int64_t(1) << 16;
constexpr int kHistBins = 2048;
constexpr int kPasses = 3;
constexpr int kPassShift[kPasses] = {21, 10, 0};
constexpr int kPassWidth[kPasses] = {11, 11, 10};
constexpr size_t kMergeAlign = 256;

struct MTensor {
  const void* theta0;
  void* out;
  int64_t numel;
  int64_t elem_offset;
  uint32_t tid, flags, t_hi, t_lo;
  int32_t dtype, pad;
};

struct MArgs {
  const MTensor* tensors;
  const Chunk* chunks;
  const void* const* experts;  // [tensor * K + e]
  uint32_t* thr;               // [tensor * K + e] TIES threshold keys
  uint32_t* prefix;            // radix select: the digits decided so far
  int64_t* rank;               // radix select: rank among keys with that prefix (1 = largest)
  unsigned long long* hist;    // [(tensor * K + e) * kHistBins]
  int64_t n_chunks;
  RoundKeys key;
  int32_t K, method;
  float gamma, c;              // c: per-expert coefficient (WA 1/K, TA gamma, DARE gamma / p_keep)
  int32_t shift, width;        // current radix pass
  uint32_t decided;            // mask of the key bits decided before this pass
  int32_t last_pass;
};

__device__ __forceinline__ uint32_t abs_key(float x) { return __float_as_uint(x) & 0x7FFFFFFFu; }

// Expert e's contribution to a 16-element group: acc += c Delta on the
// elements whose bit is set in keep (bit k: element k).
template <int DT>
__device__ __forceinline__ void merge_acc16(float c, uint32_t keep, const Raw16<DT>& x, const Raw16<DT>& t0,
                                            float2 (&acc)[8]) {
  const float2 c2 = splat(c);
#pragma unroll
  for (int h = 0; h < 8; ++h) {
    const float2 b = t0.pair(h);
    const float2 d = sub2_rn(x.pair(h), b);
    const float2 f = fma2_rn(c2, d, acc[h]);
    acc[h] = make_float2(((keep >> (2 * h)) & 1u) ? f.x : acc[h].x, ((keep >> (2 * h + 1)) & 1u) ? f.y : acc[h].y);
  }
}

template <int DT>
__device__ __forceinline__ void store_merged16(const MTensor& T, int64_t i, const Raw16<DT>& t0,
                                               const float2 (&acc)[8]) {
  float out[16];
#pragma unroll
  for (int h = 0; h < 8; ++h) {
    const float2 o = add2_rn(t0.pair(h), acc[h]);
    out[2 * h] = o.x;
    out[2 * h + 1] = o.y;
  }
  store16<DT>(T.out, i, out);
}

// Experts are loaded four at a time (all four loads in flight before the
// first is used) and accumulated in index order.
constexpr int kExpertBatch = 4;

// WA / TA on one 16-element group (vector path).
template <int DT>
__device__ __forceinline__ void merge_linear16(const MArgs& m, const MTensor& T, int t, int64_t i) {
  Raw16<DT> t0;
  load16<DT>(T.theta0, i, t0);
  float2 acc[8];
#pragma unroll
  for (int h = 0; h < 8; ++h) acc[h] = splat(0.0f);
  const void* const* xp = m.experts + t * m.K;
  int e = 0;
#pragma unroll 1
  for (; e + kExpertBatch <= m.K; e += kExpertBatch) {
    Raw16<DT> x[kExpertBatch];
#pragma unroll
    for (int b = 0; b < kExpertBatch; ++b) load16<DT>(xp[e + b], i, x[b]);
#pragma unroll
    for (int b = 0; b < kExpertBatch; ++b) merge_acc16<DT>(m.c, 0xFFFFu, x[b], t0, acc);
  }
#pragma unroll 1
  for (; e < m.K; ++e) {
    Raw16<DT> x;
    load16<DT>(xp[e], i, x);
    merge_acc16<DT>(m.c, 0xFFFFu, x, t0, acc);
  }
  store_merged16<DT>(T, i, t0, acc);
}

// DARE keep masks. A warp first draws the masks of its 32 groups for all K
// experts (expert e's mask is the Mask stream at step e) into shared memory,
// as byte masks: byte b of word q of (expert e, thread t) is 0xFF iff element
// 4q + b of t's group is kept. An element whose mask byte equals the
// threshold's high byte (probability 1/256 per element and expert) is decided
// by its low 24 bits (MASK_LO stream): these ties are queued per warp across
// all experts and then drawn by the whole warp, one MASK_LO block per lane, so
// a warp spends about one Philox pass per group on them instead of one mostly
// idle pass per expert. A queue that fills up (about K/16 ties per thread are
// expected, the capacity is 4 per thread) makes the owner draw the rest itself.
constexpr int kDareQueue = 128;
struct DareQueue {
  uint16_t q[kBlock / 32][kDareQueue];  // (lane << 8) | (expert << 4) | element
  int n[kBlock / 32];
};
// Dynamic shared memory of the DARE kernel: the queue, then uint4 keep masks
// [K][kBlock] (16 bytes per expert and thread).
constexpr size_t kDareQueueBytes = (sizeof(DareQueue) + 15) / 16 * 16;
size_t dare_smem_bytes(int K) { return kDareQueueBytes + (size_t)K * kBlock * sizeof(uint4); }

struct DareShared {
  DareQueue* qs;
  uint4* keep;  // keep[e * kBlock + thread]
};

// Byte masks of expert e from its Mask block w; ties go to the warp's queue,
// or are drawn here once the queue is full.
template <int R>
__device__ __forceinline__ uint4 dare_keep_masks(const MArgs& m, const MTensor& T, const uint4& w, int e,
                                                 uint64_t g0, DareShared& s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t kw[4];
  if (keep_bytes16(w, T.t_hi, kw) && T.t_lo != 0u) {
    uint32_t tb = tie_bits16(w, T.t_hi);
    int slot = atomicAdd(&s.qs->n[warp], __popc(tb));
    while (tb) {
      const int k = __ffs(tb) - 1;
      tb &= tb - 1u;
      if (slot < kDareQueue) {
        s.qs->q[warp][slot] = (uint16_t)((lane << 8) | (e << 4) | k);
      } else {
        const uint64_t g = g0 + (uint64_t)k;
        const uint4 l = stream_block_at<R>(m.key, (uint32_t)e, S_MASK_LO, T.tid, g >> 2);
        if ((pick(l, (unsigned)(g & 3)) >> 8) < T.t_lo) set_kept(kw, k);
      }
      ++slot;
    }
  }
  // flag bit 7 of each byte -> 0x00 / 0xFF
  return make_uint4((kw[0] >> 7) * 0xFFu, (kw[1] >> 7) * 0xFFu, (kw[2] >> 7) * 0xFFu, (kw[3] >> 7) * 0xFFu);
}

// Called by all 32 lanes of the warp (full: this lane has a vector group at
// element index g0; gw0: lane 0's group). Two experts' Mask blocks are drawn
// together (two independent Philox chains per thread). On return the lane's
// keep masks are complete.
template <int R>
__device__ __forceinline__ void dare_masks(const MArgs& m, const MTensor& T, bool full, uint64_t g0, uint64_t gw0,
                                           DareShared& s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) s.qs->n[warp] = 0;
  __syncwarp();
  if (full) {
#pragma unroll 1
    for (int e = 0; e < m.K; e += 2) {
      const uint4 w0 = stream_block_at<R>(m.key, (uint32_t)e, S_MASK, T.tid, g0 >> 4);
      const uint4 w1 = stream_block_at<R>(m.key, (uint32_t)e + 1u, S_MASK, T.tid, g0 >> 4);
      s.keep[e * kBlock + threadIdx.x] = dare_keep_masks<R>(m, T, w0, e, g0, s);
      if (e + 1 < m.K) s.keep[(e + 1) * kBlock + threadIdx.x] = dare_keep_masks<R>(m, T, w1, e + 1, g0, s);
    }
  }
  __syncwarp();
  const int n = min(s.qs->n[warp], kDareQueue);
  for (int j = lane; j < n; j += 32) {
    const uint32_t it = s.qs->q[warp][j];
    const int owner = (int)(it >> 8), e = (int)((it >> 4) & 15u), k = (int)(it & 15u);
    const uint64_t g = gw0 + 16 * (uint64_t)owner + (uint64_t)k;
    const uint4 l = stream_block_at<R>(m.key, (uint32_t)e, S_MASK_LO, T.tid, g >> 2);
    if ((pick(l, (unsigned)(g & 3)) >> 8) < T.t_lo) {
      uint32_t* kwp = reinterpret_cast<uint32_t*>(&s.keep[e * kBlock + (warp << 5) + owner]);
      atomicOr(kwp + (k >> 2), 0xFFu << (8 * (k & 3)));
    }
  }
  __syncwarp();
}

// Expert e's DARE contribution to a bf16 group: the expert's bf16 words are
// blended with theta0's by the keep masks (a dropped element takes theta0's
// bits), so a dropped element's Delta is fl(theta0 - theta0) = +0 and its
// multiply-add leaves acc unchanged (acc is never -0: it starts at +0 and a
// sum rounds to -0 only from two -0). This is exact while theta0 is finite;
// the caller takes the select path below for a group with an infinite or NaN
// theta0 (whose Delta would be NaN instead of unused).
__device__ __forceinline__ void dare_acc16_blend(float c, const uint4& km, const Raw16<DT_BF16>& x,
                                                 const Raw16<DT_BF16>& t0, float2 (&acc)[8]) {
  const float2 c2 = splat(c);
  const uint32_t kmw[4] = {km.x, km.y, km.z, km.w};
#pragma unroll
  for (int h = 0; h < 8; ++h) {
    // 16-bit lanes of the word's two elements: bytes 0, 1 (even h) or 2, 3 (odd h) of mask word h / 2
    const uint32_t lm = __byte_perm(kmw[h >> 1], 0u, (h & 1) ? 0x3322u : 0x1100u);
    const uint32_t xw = (x.r[h] & lm) | (t0.r[h] & ~lm);
    const float2 b = t0.pair(h);
    const float2 d = sub2_rn(make_float2(__uint_as_float(xw << 16), __uint_as_float(xw & 0xFFFF0000u)), b);
    acc[h] = fma2_rn(c2, d, acc[h]);
  }
}

// The same with a select per element after the multiply-add (fp32 groups, and
// bf16 groups whose theta0 is not finite).
template <int DT>
__device__ __forceinline__ void dare_acc16_select(float c, const uint4& km, const Raw16<DT>& x, const Raw16<DT>& t0,
                                                  float2 (&acc)[8]) {
  const float2 c2 = splat(c);
  const uint32_t kw[4] = {km.x, km.y, km.z, km.w};
#pragma unroll
  for (int h = 0; h < 8; ++h) {
    const float2 b = t0.pair(h);
    const float2 d = sub2_rn(x.pair(h), b);
    const float2 f = fma2_rn(c2, d, acc[h]);
    acc[h] = make_float2(kept_of(kw, 2 * h) ? f.x : acc[h].x, kept_of(kw, 2 * h + 1) ? f.y : acc[h].y);
  }
}

// Some element of a bf16 group is infinite or NaN (exponent all ones).
__device__ __forceinline__ bool nonfinite16(const Raw16<DT_BF16>& v) {
  uint32_t nf = 0u;
#pragma unroll
  for (int h = 0; h < 8; ++h) nf |= (v.r[h] & 0x7F807F80u) + 0x00800080u;  // 0x8000 in a half iff its exponent is 0xFF
  return (nf & 0x80008000u) != 0u;
}

// Experts loaded before the keep masks are drawn (fp32 groups are twice the
// registers: two, so that nothing spills).
template <int DT>
constexpr int kDarePrefetch = DT == DT_BF16 ? kExpertBatch : 2;

// DARE + TA on one 16-element group whose t0 and first kDarePrefetch experts
// are already loaded; keep masks from shared memory (masked) or all kept.
template <int DT>
__device__ __forceinline__ void dare_linear16(const MArgs& m, const MTensor& T, int t, int64_t i, bool masked,
                                              const Raw16<DT>& t0, Raw16<DT> (&x)[kExpertBatch],
                                              const DareShared& s) {
  float2 acc[8];
#pragma unroll
  for (int h = 0; h < 8; ++h) acc[h] = splat(0.0f);
  const void* const* xp = m.experts + t * m.K;
  bool blend = false;
  if (DT == DT_BF16) blend = !nonfinite16(*reinterpret_cast<const Raw16<DT_BF16>*>(&t0));
#pragma unroll 1
  for (int e = 0; e < m.K; e += kExpertBatch) {
#pragma unroll
    for (int b = 0; b < kExpertBatch; ++b)
      if ((e > 0 || b >= kDarePrefetch<DT>) && e + b < m.K) load16<DT>(xp[e + b], i, x[b]);
#pragma unroll
    for (int b = 0; b < kExpertBatch; ++b) {
      if (e + b < m.K) {
        const uint4 km = masked ? s.keep[(e + b) * kBlock + threadIdx.x]
                                : make_uint4(0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu);
        if (DT == DT_BF16 && blend)
          dare_acc16_blend(m.c, km, *reinterpret_cast<const Raw16<DT_BF16>*>(&x[b]),
                           *reinterpret_cast<const Raw16<DT_BF16>*>(&t0), acc);
        else
          dare_acc16_select<DT>(m.c, km, x[b], t0, acc);
      }
    }
  }
  store_merged16<DT>(T, i, t0, acc);
}

// TIES on one 16-element group: elect, then the disjoint mean (the experts
// are read twice; the second read is served by the L2). The oracle's
// agreement test, abs(Delta) >= thr and (sum > 0 and Delta > 0 or sum < 0 and
// Delta < 0), is taken as: key in [max(thr, 1), key(+inf)] (Delta nonzero,
// not NaN) and equal sign bits of Delta and sum; elements whose sum is 0 or
// NaN, where the oracle finds no agreeing expert, are set to 0 at the end.
template <int DT>
__device__ __forceinline__ void merge_ties16(const MArgs& m, const MTensor& T, int t, int64_t i) {
  Raw16<DT> t0;
  load16<DT>(T.theta0, i, t0);
  const void* const* xp = m.experts + t * m.K;
  const uint32_t* tp = m.thr + t * m.K;
  float sum[16];
#pragma unroll
  for (int k = 0; k < 16; ++k) sum[k] = 0.0f;
  auto elect = [&](const Raw16<DT>& x, uint32_t thr) {
#pragma unroll
    for (int h = 0; h < 8; ++h) {
      const float2 b = t0.pair(h);
      const float2 d = sub2_rn(x.pair(h), b);
      if (abs_key(d.x) >= thr) sum[2 * h] = __fadd_rn(sum[2 * h], d.x);
      if (abs_key(d.y) >= thr) sum[2 * h + 1] = __fadd_rn(sum[2 * h + 1], d.y);
    }
  };
  int e = 0;
#pragma unroll 1
  for (; e + kExpertBatch <= m.K; e += kExpertBatch) {
    Raw16<DT> x[kExpertBatch];
#pragma unroll
    for (int b = 0; b < kExpertBatch; ++b) load16<DT>(xp[e + b], i, x[b]);
#pragma unroll
    for (int b = 0; b < kExpertBatch; ++b) elect(x[b], tp[e + b]);
  }
#pragma unroll 1
  for (; e < m.K; ++e) {
    Raw16<DT> x;
    load16<DT>(xp[e], i, x);
    elect(x, tp[e]);
  }
  float part[16];
  uint32_t cnt[4] = {0u, 0u, 0u, 0u};  // four 8-bit counts per word (K <= 16)
#pragma unroll
  for (int k = 0; k < 16; ++k) part[k] = 0.0f;
  constexpr uint32_t kInfKey = 0x7F800000u;
  auto agree = [&](float d, uint32_t lo, int k) {
    const uint32_t key = abs_key(d);
    return key >= lo && key <= kInfKey && ((__float_as_uint(d) ^ __float_as_uint(sum[k])) & 0x80000000u) == 0u;
  };
  auto gather = [&](const Raw16<DT>& x, uint32_t thr) {
    const uint32_t lo = thr > 1u ? thr : 1u;
#pragma unroll
    for (int h = 0; h < 8; ++h) {
      const float2 b = t0.pair(h);
      const float2 d = sub2_rn(x.pair(h), b);
      if (agree(d.x, lo, 2 * h)) {
        part[2 * h] = __fadd_rn(part[2 * h], d.x);
        cnt[h >> 1] += 1u << (16 * (h & 1));
      }
      if (agree(d.y, lo, 2 * h + 1)) {
        part[2 * h + 1] = __fadd_rn(part[2 * h + 1], d.y);
        cnt[h >> 1] += 1u << (16 * (h & 1) + 8);
      }
    }
  };
  e = 0;
#pragma unroll 1
  for (; e + kExpertBatch <= m.K; e += kExpertBatch) {
    Raw16<DT> x[kExpertBatch];
#pragma unroll
    for (int b = 0; b < kExpertBatch; ++b) load16<DT>(xp[e + b], i, x[b]);
#pragma unroll
    for (int b = 0; b < kExpertBatch; ++b) gather(x[b], tp[e + b]);
  }
#pragma unroll 1
  for (; e < m.K; ++e) {
    Raw16<DT> x;
    load16<DT>(xp[e], i, x);
    gather(x, tp[e]);
  }
  float out[16];
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const uint32_t n = (cnt[k >> 2] >> (8 * (k & 3))) & 0xFFu;
    const bool elected = sum[k] > 0.0f || sum[k] < 0.0f;
    const float merged = (n && elected) ? __fdiv_rn(part[k], (float)n) : 0.0f;
    out[k] = __fadd_rn(t0.at(k), __fmul_rn(m.gamma, merged));
  }
  store16<DT>(T.out, i, out);
}

// Any method, one element (any alignment).
template <int R, int DT, int METHOD>
__device__ __forceinline__ void merge_elem(const MArgs& m, const MTensor& T, int t, int64_t i) {
  const float t0 = load1<DT>(T.theta0, i);
  const uint64_t g = (uint64_t)(T.elem_offset + i);
  float acc = 0.0f;
  if (METHOD == SMAT_MERGE_TIES) {
    float sum = 0.0f, part = 0.0f;
    int n = 0;
    for (int e = 0; e < m.K; ++e) {
      const float d = __fsub_rn(load1<DT>(m.experts[t * m.K + e], i), t0);
      if (abs_key(d) >= m.thr[t * m.K + e]) sum = __fadd_rn(sum, d);
    }
    for (int e = 0; e < m.K; ++e) {
      const float d = __fsub_rn(load1<DT>(m.experts[t * m.K + e], i), t0);
      if (abs_key(d) >= m.thr[t * m.K + e] && ((sum > 0.0f && d > 0.0f) || (sum < 0.0f && d < 0.0f))) {
        part = __fadd_rn(part, d);
        ++n;
      }
    }
    acc = __fmul_rn(m.gamma, n ? __fdiv_rn(part, (float)n) : 0.0f);
  } else {
    for (int e = 0; e < m.K; ++e) {
      const float d = __fsub_rn(load1<DT>(m.experts[t * m.K + e], i), t0);
      const bool kept = METHOD != SMAT_MERGE_DARE_TA || !(T.flags & TF_MASK) ||
                        elem_kept_at<R>(m.key, (uint32_t)e, T.tid, T.t_hi, T.t_lo, g);
      if (kept) acc = __fmaf_rn(m.c, d, acc);
    }
  }
  store1<DT>(T.out, i, __fadd_rn(t0, acc));
}

template <int R, int DT, int METHOD>
__global__ void __launch_bounds__(kBlock, 2) merge_kernel(const __grid_constant__ MArgs m) {
  for (int64_t ci = blockIdx.x; ci < m.n_chunks; ci += gridDim.x) {
    const Chunk ch = m.chunks[ci];
    const MTensor& T = m.tensors[ch.tensor];
    const bool vec = (T.flags & TF_VEC) != 0u;
    for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += 16 * (int64_t)kBlock) {
      if (vec && i + 16 <= ch.end) {
        if (METHOD == SMAT_MERGE_TIES)
          merge_ties16<DT>(m, T, ch.tensor, i);
        else
          merge_linear16<DT>(m, T, ch.tensor, i);
      } else {
        const int64_t e_end = (i + 16 < ch.end) ? i + 16 : ch.end;
        for (int64_t e = i; e < e_end; ++e) merge_elem<R, DT, METHOD>(m, T, ch.tensor, e);
      }
    }
  }
}

// DARE + TA. The loop runs the same number of iterations on every lane of
// the CTA (the keep masks are drawn warp-cooperatively); t0 and the first
// experts are loaded before the masks are drawn, so the loads are in flight
// during the Philox work.
template <int R, int DT>
__global__ void __launch_bounds__(kBlock, 2) dare_kernel(const __grid_constant__ MArgs m) {
  extern __shared__ __align__(16) unsigned char dare_smem[];
  DareShared s;
  s.qs = reinterpret_cast<DareQueue*>(dare_smem);
  s.keep = reinterpret_cast<uint4*>(dare_smem + kDareQueueBytes);
  const int warp = threadIdx.x >> 5;
  for (int64_t ci = blockIdx.x; ci < m.n_chunks; ci += gridDim.x) {
    const Chunk ch = m.chunks[ci];
    const MTensor& T = m.tensors[ch.tensor];
    const bool vec = (T.flags & TF_VEC) != 0u;
    const bool masked = (T.flags & TF_MASK) != 0u;
    const void* const* xp = m.experts + ch.tensor * m.K;
    for (int64_t base = ch.begin; base < ch.end; base += 16 * (int64_t)kBlock) {
      const int64_t i = base + 16 * (int64_t)threadIdx.x;
      const bool full = vec && i + 16 <= ch.end;
      Raw16<DT> t0, x[kExpertBatch];
      if (full) {
        load16<DT>(T.theta0, i, t0);
#pragma unroll
        for (int b = 0; b < kDarePrefetch<DT>; ++b)
          if (b < m.K) load16<DT>(xp[b], i, x[b]);
      }
      if (masked)
        dare_masks<R>(m, T, full, (uint64_t)(T.elem_offset + i),
                      (uint64_t)(T.elem_offset + base + 16 * 32 * (int64_t)warp), s);
      if (full) {
        dare_linear16<DT>(m, T, ch.tensor, i, masked, t0, x, s);
      } else if (i < ch.end) {
        const int64_t e_end = (i + 16 < ch.end) ? i + 16 : ch.end;
        for (int64_t e = i; e < e_end; ++e) merge_elem<R, DT, SMAT_MERGE_DARE_TA>(m, T, ch.tensor, e);
      }
    }
  }
}

// One radix pass of the TIES threshold selection. A work item is a chunk
// and up to kHistExperts of its experts: theta0 is read once for them, and
// each thread has theta0's and every expert's 32-byte load in flight at once;
// one shared-memory histogram per expert, flushed into the 64-bit global bins.
constexpr int kHistExperts = 4;

// The key is abs(Delta)'s bits: its sign bit is 0, so the prefix test and
// the digit are taken on Delta's raw bits with bit 31 masked out of both
// (one operation per key fewer). FIRST: the first pass, where no digit is
// decided yet and every key counts.
template <int DT, bool FIRST>
__global__ void __launch_bounds__(kBlock, DT == DT_BF16 ? 4 : 1) ties_hist_kernel(const __grid_constant__ MArgs m) {
  __shared__ uint32_t h[kHistExperts * kHistBins];
  const int nbat = (m.K + kHistExperts - 1) / kHistExperts;
  const int64_t items = m.n_chunks * nbat;
  const uint32_t digit = ((1u << m.width) - 1u) & (0x7FFFFFFFu >> m.shift);
  const uint32_t dm = m.decided & 0x7FFFFFFFu;
  for (int64_t w = blockIdx.x; w < items; w += gridDim.x) {
    const int64_t ci = w / nbat;
    const int e0 = (int)(w % nbat) * kHistExperts;
    const int ne = m.K - e0 < kHistExperts ? m.K - e0 : kHistExperts;
    const Chunk ch = m.chunks[ci];
    const MTensor& T = m.tensors[ch.tensor];
    const int slot0 = ch.tensor * m.K + e0;
    for (int b = threadIdx.x; b < kHistExperts * kHistBins; b += kBlock) h[b] = 0u;
    __syncthreads();
    uint32_t P[kHistExperts];
    const void* xp[kHistExperts];
#pragma unroll
    for (int b = 0; b < kHistExperts; ++b) {
      P[b] = b < ne ? m.prefix[slot0 + b] : 0u;
      xp[b] = b < ne ? m.experts[slot0 + b] : nullptr;
    }
    const bool vec = (T.flags & TF_VEC) != 0u;
    for (int64_t i = ch.begin + 16 * (int64_t)threadIdx.x; i < ch.end; i += 16 * (int64_t)kBlock) {
      if (vec && i + 16 <= ch.end) {
        Raw16<DT> t0, x[kHistExperts];
        load16<DT>(T.theta0, i, t0);
#pragma unroll
        for (int b = 0; b < kHistExperts; ++b)
          if (b < ne) load16<DT>(xp[b], i, x[b]);
#pragma unroll
        for (int b = 0; b < kHistExperts; ++b) {
          if (b < ne) {
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const float2 d = sub2_rn(x[b].pair(q), t0.pair(q));
              const uint32_t k0 = __float_as_uint(d.x), k1 = __float_as_uint(d.y);
              if (FIRST || (k0 & dm) == P[b]) atomicAdd(&h[b * kHistBins + ((k0 >> m.shift) & digit)], 1u);
              if (FIRST || (k1 & dm) == P[b]) atomicAdd(&h[b * kHistBins + ((k1 >> m.shift) & digit)], 1u);
            }
          }
        }
      } else {
        const int64_t e_end = (i + 16 < ch.end) ? i + 16 : ch.end;
        for (int64_t k = i; k < e_end; ++k) {
          const float t0 = load1<DT>(T.theta0, k);
          for (int b = 0; b < ne; ++b) {
            const uint32_t key = abs_key(__fsub_rn(load1<DT>(xp[b], k), t0));
            if ((key & m.decided) == P[b]) atomicAdd(&h[b * kHistBins + ((key >> m.shift) & digit)], 1u);
          }
        }
      }
    }
    __syncthreads();
    // the ne histograms are consecutive slots' bins in the global array
    unsigned long long* gh = m.hist + (size_t)slot0 * kHistBins;
    for (int b = threadIdx.x; b < ne * kHistBins; b += kBlock)
      if (h[b]) atomicAdd(gh + b, (unsigned long long)h[b]);
    __syncthreads();
  }
}

// After a pass: one CTA per (tensor, expert) picks the digit whose bin holds
// the rank-th largest key (bins scanned from the top), records it and the
// rank within that bin, and clears the histogram for the next pass.
__global__ void __launch_bounds__(kBlock) ties_select_kernel(const __grid_constant__ MArgs m) {
  __shared__ unsigned long long s_sum[kBlock];
  __shared__ int s_digit;
  __shared__ long long s_above;
  const int slot = blockIdx.x;
  unsigned long long* gh = m.hist + (size_t)slot * kHistBins;
  const long long r = m.rank[slot];
  const int nb = 1 << m.width;
  const int per = nb / kBlock;  // bins per thread, highest bins in thread 0
  unsigned long long local = 0;
  const int top = nb - 1 - threadIdx.x * per;
  for (int k = 0; k < per; ++k) local += gh[top - k];
  s_sum[threadIdx.x] = local;
  if (threadIdx.x == 0) {
    s_digit = -1;
    s_above = 0;
  }
  __syncthreads();
  // inclusive scan from the top (Hillis-Steele; 8 steps over 256 entries)
  for (int o = 1; o < kBlock; o <<= 1) {
    const unsigned long long v = threadIdx.x >= o ? s_sum[threadIdx.x - o] : 0ull;
    __syncthreads();
    s_sum[threadIdx.x] += v;
    __syncthreads();
  }
  const unsigned long long incl = s_sum[threadIdx.x];
  const unsigned long long excl = incl - local;
  if (r > 0 && (long long)excl < r && r <= (long long)incl) {
    unsigned long long acc = excl;
    for (int k = 0; k < per; ++k) {
      const unsigned long long c = gh[top - k];
      if ((long long)(acc + c) >= r) {
        s_digit = top - k;
        s_above = (long long)acc;
        break;
      }
      acc += c;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && r > 0 && s_digit >= 0) {
    const uint32_t p = m.prefix[slot] | ((uint32_t)s_digit << m.shift);
    m.prefix[slot] = p;
    m.rank[slot] = r - s_above;
    if (m.last_pass) m.thr[slot] = p;
  }
  for (int b = threadIdx.x; b < kHistBins; b += kBlock) gh[b] = 0ull;
}

template <int R, int DT>
cudaError_t merge_method(const MArgs& m, int grid, cudaStream_t s) {
  switch (m.method) {
    case SMAT_MERGE_WA: merge_kernel<R, DT, SMAT_MERGE_WA><<<grid, kBlock, 0, s>>>(m); break;
    case SMAT_MERGE_TA: merge_kernel<R, DT, SMAT_MERGE_TA><<<grid, kBlock, 0, s>>>(m); break;
    case SMAT_MERGE_DARE_TA: {
      const size_t smem = dare_smem_bytes(m.K);
      if (smem > 48 * 1024) {
        const cudaError_t e = cudaFuncSetAttribute(dare_kernel<R, DT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   (int)smem);
        if (e != cudaSuccess) return e;
      }
      dare_kernel<R, DT><<<grid, kBlock, smem, s>>>(m);
      break;
    }
    default: merge_kernel<R, DT, SMAT_MERGE_TIES><<<grid, kBlock, 0, s>>>(m); break;
  }
  return cudaGetLastError();
}

// ------------------------------------------------------------------- host ---
struct MLayout {
  size_t tensors, chunks, experts, thr, prefix, rank, hist, total;
};

size_t align_m(size_t x) { return (x + kMergeAlign - 1) / kMergeAlign * kMergeAlign; }

MLayout merge_layout(int32_t n, int64_t n_chunks, int K, bool ties) {
  MLayout L;
  size_t off = 0;
  const size_t slots = (size_t)n * (size_t)K;
  L.tensors = off; off = align_m(off + sizeof(MTensor) * (size_t)n);
  L.chunks = off;  off = align_m(off + sizeof(Chunk) * (size_t)n_chunks);
  L.experts = off; off = align_m(off + sizeof(void*) * slots);
  L.thr = off;     off = align_m(off + sizeof(uint32_t) * slots);
  L.prefix = off;  off = align_m(off + sizeof(uint32_t) * slots);
  L.rank = off;    off = align_m(off + sizeof(int64_t) * slots);
  L.hist = off;    off = align_m(off + (ties ? sizeof(unsigned long long) * kHistBins * slots : 0));
  L.total = off;
  return L;
}

smat_status mfail(smat_status s, const char* fmt, ...) {
  char buf[256];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  return (smat_status)record_error_code((int)s, buf);
}

bool m_overlaps(const void* a, size_t na, const void* b, size_t nb) {
  const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
  return x < y + nb && y < x + na;
}

// Host-side validation (no device access); returns the chunk count and the
// list's dtype (one dtype per call).
smat_status merge_check(const smat_merge_tensor* t, int32_t n, const smat_merge_config* cfg, int64_t* n_chunks,
                        int32_t* dtype_out) {
  if (!cfg) return mfail(SMAT_ERR_INVALID_ARG, "cfg is NULL");
  if (cfg->method < SMAT_MERGE_WA || cfg->method > SMAT_MERGE_TIES)
    return mfail(SMAT_ERR_UNSUPPORTED, "merge method %d not supported", cfg->method);
  if (cfg->n_experts < 1 || cfg->n_experts > kMergeMaxExperts)
    return mfail(SMAT_ERR_INVALID_ARG, "n_experts %d not in [1, %d]", cfg->n_experts, kMergeMaxExperts);
  if (!std::isfinite(cfg->gamma)) return mfail(SMAT_ERR_INVALID_ARG, "gamma not finite");
  if (!(cfg->p_drop >= 0.0f && cfg->p_drop < 1.0f)) return mfail(SMAT_ERR_INVALID_ARG, "p_drop not in [0, 1)");
  if (!(cfg->retention > 0.0f && cfg->retention <= 1.0f))
    return mfail(SMAT_ERR_INVALID_ARG, "retention not in (0, 1]");
  if (cfg->philox_rounds != 0 && cfg->philox_rounds != 7 && cfg->philox_rounds != 10)
    return mfail(SMAT_ERR_UNSUPPORTED, "philox_rounds %d not supported (7 or 10)", cfg->philox_rounds);
  if (cfg->flags != 0) return mfail(SMAT_ERR_UNSUPPORTED, "unknown flags 0x%x", cfg->flags);
  if (n < 0 || (n > 0 && !t)) return mfail(SMAT_ERR_INVALID_ARG, "bad tensor list");
  std::unordered_set<uint32_t> ids;
  int64_t nc = 0;
  for (int32_t k = 0; k < n; ++k) {
    const smat_merge_tensor& d = t[k];
    if (d.numel < 0 || d.numel >= (int64_t(1) << 40))
      return mfail(SMAT_ERR_INVALID_ARG, "tensor %d: numel out of range", k);
    if (d.elem_offset < 0 || d.elem_offset >= (int64_t(1) << 62) - d.numel)
      return mfail(SMAT_ERR_INVALID_ARG, "tensor %d: elem_offset out of range", k);
    if (d.tensor_id >= kGlobalAlphaTensor) return mfail(SMAT_ERR_INVALID_ARG, "tensor %d: tensor_id too large", k);
    if (!ids.insert(d.tensor_id).second) return mfail(SMAT_ERR_INVALID_ARG, "tensor %d: duplicate tensor_id", k);
    if (d.dtype != SMAT_F32 && d.dtype != SMAT_BF16)
      return mfail(SMAT_ERR_UNSUPPORTED, "tensor %d: dtype %d not supported", k, d.dtype);
    if (d.dtype != t[0].dtype) return mfail(SMAT_ERR_UNSUPPORTED, "tensor %d: one dtype per merge call", k);
    if (d.numel > 0) {
      const size_t es = d.dtype == SMAT_BF16 ? 2 : 4, bytes = es * (size_t)d.numel;
      if (!d.theta0 || !d.out || !d.experts) return mfail(SMAT_ERR_INVALID_ARG, "tensor %d: NULL pointer", k);
      if ((uintptr_t)d.theta0 % es || (uintptr_t)d.out % es)
        return mfail(SMAT_ERR_ALIGNMENT, "tensor %d: pointer not aligned to its element size", k);
      if (d.out != d.theta0 && m_overlaps(d.out, bytes, d.theta0, bytes))
        return mfail(SMAT_ERR_INVALID_ARG, "tensor %d: out overlaps theta0 without being equal to it", k);
      for (int e = 0; e < cfg->n_experts; ++e) {
        const void* x = d.experts[e];
        if (!x) return mfail(SMAT_ERR_INVALID_ARG, "tensor %d: expert %d is NULL", k, e);
        if ((uintptr_t)x % es) return mfail(SMAT_ERR_ALIGNMENT, "tensor %d: expert %d misaligned", k, e);
        if (m_overlaps(d.out, bytes, x, bytes))
          return mfail(SMAT_ERR_INVALID_ARG, "tensor %d: out overlaps expert %d", k, e);
      }
    }
    nc += (d.numel + kMergeChunk - 1) / kMergeChunk;
  }
  if (nc >= (int64_t(1) << 31)) return mfail(SMAT_ERR_INVALID_ARG, "too many chunks");
  *n_chunks = nc;
  *dtype_out = n > 0 ? t[0].dtype : SMAT_F32;
  return SMAT_OK;
}

template <int R, int DT>
cudaError_t merge_launch(MArgs m, int64_t slots, bool ties, int sms, cudaStream_t s) {
  if (ties) {
    const int64_t items = m.n_chunks * ((m.K + kHistExperts - 1) / kHistExperts);
    int occ = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, ties_hist_kernel<DT, false>, kBlock, 0) != cudaSuccess ||
        occ < 1)
      occ = 1;
    const int64_t resident = (int64_t)occ * sms;
    const int hgrid = (int)(items < resident ? items : resident);
    for (int p = 0; p < kPasses; ++p) {
      m.shift = kPassShift[p];
      m.width = kPassWidth[p];
      m.decided = (m.shift + m.width >= 32) ? 0u : ~((1u << (m.shift + m.width)) - 1u);
      m.last_pass = p == kPasses - 1;
      if (p == 0)
        ties_hist_kernel<DT, true><<<hgrid, kBlock, 0, s>>>(m);
      else
        ties_hist_kernel<DT, false><<<hgrid, kBlock, 0, s>>>(m);
      ties_select_kernel<<<(int)slots, kBlock, 0, s>>>(m);
    }
  }
  const int grid = (int)(m.n_chunks < 2 * (int64_t)sms ? m.n_chunks : 2 * (int64_t)sms);
  return merge_method<R, DT>(m, grid, s);
}

}  // namespace
}  // namespace smat

using namespace smat;

extern "C" size_t smat_merge_workspace_bytes(const smat_merge_tensor* tensors, int32_t n_tensors,
                                             const smat_merge_config* cfg) {
  int64_t nc = 0;
  int32_t dt = 0;
  if (merge_check(tensors, n_tensors, cfg, &nc, &dt) != SMAT_OK) return 0;
  return merge_layout(n_tensors, nc, cfg->n_experts, cfg->method == SMAT_MERGE_TIES).total;
}

extern "C" smat_status smat_merge(const smat_merge_tensor* tensors, int32_t n_tensors, const smat_merge_config* cfg,
                                  void* d_workspace, size_t workspace_bytes, smat_stream_t stream) {
  int64_t nc = 0;
  int32_t dtype = 0;
  smat_status st = merge_check(tensors, n_tensors, cfg, &nc, &dtype);
  if (st != SMAT_OK) return st;
  const int K = cfg->n_experts;
  const bool ties = cfg->method == SMAT_MERGE_TIES;
  const MLayout L = merge_layout(n_tensors, nc, K, ties);
  if (!d_workspace || (uintptr_t)d_workspace % kMergeAlign)
    return mfail(SMAT_ERR_WORKSPACE, "workspace NULL or not 256-byte aligned");
  if (workspace_bytes < L.total) return mfail(SMAT_ERR_WORKSPACE, "workspace %zu < %zu bytes", workspace_bytes, L.total);
  for (int32_t k = 0; k < n_tensors; ++k) {
    if (tensors[k].numel <= 0) continue;
    int ok = gpu_can_access(tensors[k].theta0) == 1 && gpu_can_access(tensors[k].out) == 1;
    for (int e = 0; ok && e < K; ++e) ok = gpu_can_access(tensors[k].experts[e]) == 1;
    if (!ok) return mfail(SMAT_ERR_INVALID_ARG, "tensor %d: a pointer is not accessible from the GPU", k);
  }
  if (n_tensors == 0 || nc == 0) return SMAT_OK;

  // tables (host), then one upload each
  const float keep = 1.0f - cfg->p_drop;
  const uint64_t T = (uint64_t)std::floor((double)keep * 4294967296.0);
  std::vector<MTensor> ht((size_t)n_tensors);
  std::vector<Chunk> hc;
  hc.reserve((size_t)nc);
  std::vector<const void*> hx((size_t)n_tensors * (size_t)K, nullptr);
  std::vector<int64_t> hrank((size_t)n_tensors * (size_t)K, 0);
  for (int32_t k = 0; k < n_tensors; ++k) {
    const smat_merge_tensor& d = tensors[k];
    MTensor& M = ht[(size_t)k];
    std::memset(&M, 0, sizeof(M));
    M.theta0 = d.theta0;
    M.out = d.out;
    M.numel = d.numel;
    M.elem_offset = d.elem_offset;
    M.tid = d.tensor_id;
    M.dtype = d.dtype;
    bool vec = d.numel > 0 && (uintptr_t)d.theta0 % 32 == 0 && (uintptr_t)d.out % 32 == 0 && d.elem_offset % 16 == 0;
    for (int e = 0; e < K; ++e) {
      hx[(size_t)k * K + e] = d.numel > 0 ? d.experts[e] : nullptr;
      vec = vec && (uintptr_t)d.experts[e] % 32 == 0;
    }
    M.flags = vec ? TF_VEC : 0u;
    if (cfg->method == SMAT_MERGE_DARE_TA && T < (uint64_t(1) << 32)) {
      M.flags |= TF_MASK;
      M.t_hi = (uint32_t)(T >> 24);
      M.t_lo = (uint32_t)(T & 0xFFFFFFu);
    }
    if (ties && d.numel > 0) {
      int64_t r = (int64_t)std::ceil((double)cfg->retention * (double)d.numel);
      r = r < 1 ? 1 : (r > d.numel ? d.numel : r);
      for (int e = 0; e < K; ++e) hrank[(size_t)k * K + e] = r;
    }
    for (int64_t j = 0; j * kMergeChunk < d.numel; ++j) {
      Chunk ch;
      ch.tensor = k;
      ch.pad = 0;
      ch.begin = j * kMergeChunk;
      ch.end = (j + 1) * kMergeChunk < d.numel ? (j + 1) * kMergeChunk : d.numel;
      hc.push_back(ch);
    }
  }
  char* ws = static_cast<char*>(d_workspace);
  MArgs m;
  std::memset(&m, 0, sizeof(m));
  m.tensors = reinterpret_cast<const MTensor*>(ws + L.tensors);
  m.chunks = reinterpret_cast<const Chunk*>(ws + L.chunks);
  m.experts = reinterpret_cast<const void* const*>(ws + L.experts);
  m.thr = reinterpret_cast<uint32_t*>(ws + L.thr);
  m.prefix = reinterpret_cast<uint32_t*>(ws + L.prefix);
  m.rank = reinterpret_cast<int64_t*>(ws + L.rank);
  m.hist = ties ? reinterpret_cast<unsigned long long*>(ws + L.hist) : nullptr;
  m.n_chunks = nc;
  m.key = make_round_keys(cfg->seed);
  m.K = K;
  m.method = cfg->method;
  m.gamma = cfg->gamma;
  const float inv_keep = (float)(1.0 / (double)keep);
  m.c = cfg->method == SMAT_MERGE_WA ? (float)(1.0 / (double)K)
        : cfg->method == SMAT_MERGE_DARE_TA ? cfg->gamma * inv_keep : cfg->gamma;
  const size_t slots = (size_t)n_tensors * (size_t)K;
  cudaError_t e = cudaMemcpyAsync(ws + L.tensors, ht.data(), sizeof(MTensor) * ht.size(), cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess) e = cudaMemcpyAsync(ws + L.chunks, hc.data(), sizeof(Chunk) * hc.size(), cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess) e = cudaMemcpyAsync(ws + L.experts, hx.data(), sizeof(void*) * slots, cudaMemcpyHostToDevice, stream);
  if (e != cudaSuccess) return mfail(SMAT_ERR_CUDA, "merge table upload failed");
  int dev = 0, sms = 1;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return mfail(SMAT_ERR_CUDA, "device query failed");
  const int rounds = cfg->philox_rounds == 7 ? 7 : 10;
  if (ties) {
    e = cudaMemsetAsync(ws + L.prefix, 0, sizeof(uint32_t) * slots, stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(ws + L.thr, 0, sizeof(uint32_t) * slots, stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(ws + L.hist, 0, sizeof(unsigned long long) * kHistBins * slots, stream);
    if (e == cudaSuccess) e = cudaMemcpyAsync(ws + L.rank, hrank.data(), sizeof(int64_t) * slots, cudaMemcpyHostToDevice, stream);
    if (e != cudaSuccess) return mfail(SMAT_ERR_CUDA, "TIES state initialisation failed");
  }
  const int64_t slots64 = (int64_t)slots;
  if (dtype == SMAT_BF16)
    e = rounds == 7 ? merge_launch<7, DT_BF16>(m, slots64, ties, sms, stream)
                    : merge_launch<10, DT_BF16>(m, slots64, ties, sms, stream);
  else
    e = rounds == 7 ? merge_launch<7, DT_F32>(m, slots64, ties, sms, stream)
                    : merge_launch<10, DT_F32>(m, slots64, ties, sms, stream);
  if (e != cudaSuccess) return mfail(SMAT_ERR_CUDA, "merge launch failed");
  return SMAT_OK;
}

extern "C" smat_status smat_merge_ties_thresholds(const smat_merge_tensor* tensors, int32_t n_tensors,
                                                  const smat_merge_config* cfg, const void* d_workspace,
                                                  uint32_t* d_out, smat_stream_t stream) {
  int64_t nc = 0;
  int32_t dtype = 0;
  smat_status st = merge_check(tensors, n_tensors, cfg, &nc, &dtype);
  if (st != SMAT_OK) return st;
  if (cfg->method != SMAT_MERGE_TIES) return mfail(SMAT_ERR_STATE, "not a TIES configuration");
  if (!d_workspace || !d_out) return mfail(SMAT_ERR_INVALID_ARG, "NULL pointer");
  const MLayout L = merge_layout(n_tensors, nc, cfg->n_experts, true);
  const size_t bytes = sizeof(uint32_t) * (size_t)n_tensors * (size_t)cfg->n_experts;
  if (bytes && cudaMemcpyAsync(d_out, static_cast<const char*>(d_workspace) + L.thr, bytes,
                               cudaMemcpyDeviceToDevice, stream) != cudaSuccess)
    return mfail(SMAT_ERR_CUDA, "threshold copy failed");
  return SMAT_OK;
}
