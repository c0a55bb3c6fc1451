// Host side of libsmat: argument validation, device tables, launches.
// The C ABI is declared in include/smat.h.

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <unordered_set>
#include <vector>

#include <cuda_runtime.h>

#include "smat.h"
#include "smat_internal.h"

using namespace smat;

namespace {

thread_local std::string g_last_error;

smat_status fail(smat_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  std::vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

smat_status cuda_fail(cudaError_t e, const char* what) {
  return fail(SMAT_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

constexpr size_t kAlign = 256;
size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }
size_t elem_size(int32_t dt) { return dt == SMAT_BF16 ? 2 : 4; }
constexpr int64_t kMaxNumel = int64_t(1) << 40;

struct Layout {
  size_t tensors, chunks, scal, partials, grads, items, sync, total;
};

// sync region: work counters (kMaxRanges), error flag, pad, then per tensor
// tensor_done and ready.
size_t sync_words(int32_t n) { return 4 + 2 * (size_t)n; }

int64_t chunks_of(int64_t numel, int64_t chunk_elems) { return (numel + chunk_elems - 1) / chunk_elems; }

// The work-chunk size of a list: the largest power of two cs in
// [kMinChunkElems, kMaxChunkElems] with cs^2 / 64 <= total elements (a pure
// function of the list and flags, so the workspace size and the context
// agree).
int64_t chunk_elems_for(const smat_tensor_desc* t, int32_t n, const smat_config* cfg) {
  const int forced = (cfg->flags & SMAT_FLAG_CHUNK_LOG2_MASK) >> 8;
  if (forced) return int64_t(1) << forced;
  int64_t total = 0;
  for (int32_t k = 0; k < n; ++k) total = std::min(total + t[k].numel, int64_t(1) << 62);
  int64_t cs = kMinChunkElems;
  while (cs < kMaxChunkElems && (2 * cs) * (2 * cs) / 64 <= total) cs *= 2;
  return cs;
}

Layout layout_for(int32_t n, int64_t n_chunks, bool any_sigma_rel) {
  Layout L;
  size_t off = 0;
  L.tensors = off; off = align_up(off + sizeof(DevTensor) * (size_t)n);
  L.chunks = off;  off = align_up(off + sizeof(Chunk) * (size_t)n_chunks);
  L.scal = off;    off = align_up(off + sizeof(DevScalars) * (size_t)n);
  L.partials = off; off = align_up(off + (any_sigma_rel ? sizeof(StatPartial) * (size_t)n_chunks : 0));
  // the gradient-map and fused-AdamW pointer tables share this region
  L.grads = off;   off = align_up(off + std::max(sizeof(GradPtr), sizeof(AdamPtr)) * (size_t)n);
  L.items = off;   off = align_up(off + sizeof(int32_t) * (any_sigma_rel ? 2 : 1) * (size_t)n_chunks);
  L.sync = off;    off = align_up(off + sizeof(int32_t) * sync_words(n));
  L.total = off;
  return L;
}

bool finite(float x) { return std::isfinite(x); }

smat_status check_config(const smat_config* cfg) {
  if (!cfg) return fail(SMAT_ERR_INVALID_ARG, "cfg is NULL");
  if (cfg->alpha_mode < SMAT_ALPHA_GLOBAL || cfg->alpha_mode > SMAT_ALPHA_PER_ELEMENT)
    return fail(SMAT_ERR_UNSUPPORTED, "alpha_mode %d not supported", cfg->alpha_mode);
  if (cfg->noise != SMAT_NOISE_UNIFORM && cfg->noise != SMAT_NOISE_GAUSSIAN && cfg->noise != SMAT_NOISE_LAPLACE)
    return fail(SMAT_ERR_UNSUPPORTED, "noise %d not supported", cfg->noise);
  if (cfg->noise == SMAT_NOISE_LAPLACE && cfg->philox_rounds == 7)
    return fail(SMAT_ERR_UNSUPPORTED, "Laplace noise is built for 10 Philox rounds");
  if (cfg->philox_rounds != 0 && cfg->philox_rounds != 7 && cfg->philox_rounds != 10)
    return fail(SMAT_ERR_UNSUPPORTED, "philox_rounds %d not supported (7 or 10)", cfg->philox_rounds);
  if (cfg->draw_bits != 0 && cfg->draw_bits != 16 && cfg->draw_bits != 32)
    return fail(SMAT_ERR_UNSUPPORTED, "draw_bits %d not supported (32 or 16)", cfg->draw_bits);
  if (cfg->flags & ~(SMAT_FLAG_UNFUSED_STATS | SMAT_FLAG_CHUNK_LOG2_MASK))
    return fail(SMAT_ERR_UNSUPPORTED, "unknown flags 0x%x", cfg->flags);
  const int chunk_log2 = (cfg->flags & SMAT_FLAG_CHUNK_LOG2_MASK) >> 8;
  if (chunk_log2 != 0 && (chunk_log2 < 12 || chunk_log2 > 18))
    return fail(SMAT_ERR_UNSUPPORTED, "chunk log2 %d not in [12, 18]", chunk_log2);
  if (!finite(cfg->alpha_min) || !finite(cfg->alpha_max) || cfg->alpha_min > cfg->alpha_max)
    return fail(SMAT_ERR_INVALID_ARG, "alpha range [%g, %g) invalid", cfg->alpha_min, cfg->alpha_max);
  return SMAT_OK;
}

bool overlaps(const void* a, size_t abytes, const void* b, size_t bbytes) {
  const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
  return x < y + bbytes && y < x + abytes;
}

smat_status check_tensors(const smat_tensor_desc* t, int32_t n, const smat_config* cfg, int64_t* n_chunks,
                          bool* any_rel, int64_t* chunk_elems) {
  if (n < 0) return fail(SMAT_ERR_INVALID_ARG, "n_tensors %d < 0", n);
  if (n > 0 && !t) return fail(SMAT_ERR_INVALID_ARG, "tensors is NULL");
  std::unordered_set<uint32_t> ids;
  int64_t nc = 0;
  bool rel = false;
  for (int32_t k = 0; k < n; ++k) {
    const smat_tensor_desc& d = t[k];
    if (d.numel < 0 || d.numel >= kMaxNumel)
      return fail(SMAT_ERR_INVALID_ARG, "tensor %d: numel %lld out of range", k, (long long)d.numel);
    if (d.elem_offset < 0 || d.elem_offset >= (int64_t(1) << 62) - d.numel)
      return fail(SMAT_ERR_INVALID_ARG, "tensor %d: elem_offset %lld out of range", k, (long long)d.elem_offset);
    if (d.tensor_id >= kGlobalAlphaTensor)
      return fail(SMAT_ERR_INVALID_ARG, "tensor %d: tensor_id %u >= 0x0FFFFFFF", k, d.tensor_id);
    if (!ids.insert(d.tensor_id).second)
      return fail(SMAT_ERR_INVALID_ARG, "tensor %d: duplicate tensor_id %u", k, d.tensor_id);
    if (d.dtype != SMAT_F32 && d.dtype != SMAT_BF16)
      return fail(SMAT_ERR_UNSUPPORTED, "tensor %d: dtype %d not supported", k, d.dtype);
    if (!(d.keep_prob >= 0.0f && d.keep_prob <= 1.0f))
      return fail(SMAT_ERR_INVALID_ARG, "tensor %d: keep_prob %g not in [0, 1]", k, d.keep_prob);
    if (!finite(d.sigma) || d.sigma < 0.0f)
      return fail(SMAT_ERR_INVALID_ARG, "tensor %d: sigma %g invalid", k, d.sigma);
    if (!finite(d.sigma_rel) || d.sigma_rel < 0.0f)
      return fail(SMAT_ERR_INVALID_ARG, "tensor %d: sigma_rel %g invalid", k, d.sigma_rel);
    if (d.numel > 0) {
      if (!d.theta || !d.theta0 || !d.sim)
        return fail(SMAT_ERR_INVALID_ARG, "tensor %d: NULL data pointer", k);
      const size_t es = elem_size(d.dtype);
      if ((uintptr_t)d.theta % es || (uintptr_t)d.theta0 % es || (uintptr_t)d.sim % es)
        return fail(SMAT_ERR_ALIGNMENT, "tensor %d: pointer not aligned to %zu bytes", k, es);
      const size_t bytes = es * (size_t)d.numel;
      // sim == theta0 is the in-place mode; any other overlap is an error
      if (overlaps(d.sim, bytes, d.theta, bytes) || (d.sim != d.theta0 && overlaps(d.sim, bytes, d.theta0, bytes)))
        return fail(SMAT_ERR_INVALID_ARG, "tensor %d: sim overlaps theta, or theta0 without being equal to it", k);
    }
    rel = rel || d.sigma_rel > 0.0f;
  }
  const int64_t cs = chunk_elems_for(t, n, cfg);
  for (int32_t k = 0; k < n; ++k) nc += chunks_of(t[k].numel, cs);
  *chunk_elems = cs;
  if (nc >= (int64_t(1) << 31)) return fail(SMAT_ERR_INVALID_ARG, "too many chunks (%lld)", (long long)nc);
  *n_chunks = nc;
  *any_rel = rel;
  return SMAT_OK;
}

// Every data pointer must be usable by the GPU's kernels as it is: device or
// managed memory, host memory registered with CUDA (pinned; under unified
// addressing its device address is the host address), or any host memory
// when the device reads pageable memory directly (coherent CPU-GPU systems).
smat_status check_gpu_access(const smat_tensor_desc* t, int32_t n) {
  for (int32_t k = 0; k < n; ++k) {
    if (t[k].numel <= 0) continue;
    const void* ptrs[3] = {t[k].theta, t[k].theta0, t[k].sim};
    for (const void* p : ptrs) {
      const int ok = gpu_can_access(p);
      if (ok < 0) return fail(SMAT_ERR_CUDA, "no current CUDA device or pointer attributes unavailable");
      if (!ok) return fail(SMAT_ERR_INVALID_ARG, "tensor %d: a data pointer is not accessible from the GPU", k);
    }
  }
  return SMAT_OK;
}

RoundKeys make_keys(uint64_t seed) { return make_round_keys(seed); }

}  // namespace

// 1 if the kernels can dereference p as it is: device or managed memory, host
// memory registered with CUDA (pinned; under unified addressing its device
// address is the host address), or any host memory when the device reads
// pageable memory directly (coherent CPU-GPU systems); 0 if not; -1 on a
// CUDA error.
int smat::gpu_can_access(const void* p) {
  int dev = 0, pageable = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return -1;
  if (cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccess, dev) != cudaSuccess) pageable = 0;
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return -1;
  }
  return (at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged ||
          (at.type == cudaMemoryTypeHost && at.devicePointer == p) ||
          (at.type == cudaMemoryTypeUnregistered && pageable))
             ? 1
             : 0;
}

// Philox round keys of a seed: key = (seed mod 2^32, seed div 2^32), each
// round's key advanced by the Weyl increments of the key schedule.
RoundKeys smat::make_round_keys(uint64_t seed) {
  RoundKeys k;
  uint32_t a = (uint32_t)(seed & 0xFFFFFFFFu), b = (uint32_t)(seed >> 32);
  for (int r = 0; r < kMaxRounds; ++r) {
    k.k0[r] = a;
    k.k1[r] = b;
    a += 0x9E3779B9u;
    b += 0xBB67AE85u;
  }
  return k;
}

int smat::record_error_code(int status, const char* msg) {
  g_last_error = msg;
  return status;
}

struct smat_ctx {
  std::vector<smat_tensor_desc> desc;
  smat_config cfg;
  int rounds = 10;
  std::vector<DevTensor> h_tensors;
  std::vector<Chunk> h_chunks;
  int64_t range_begin[2] = {0, 0};  // chunk range per dtype (F32, BF16)
  int64_t range_end[2] = {0, 0};
  bool any_sigma_rel = false;
  // in-place tensors (sim == theta0): their sim buffers hold theta0 until a
  // forward overwrites it; a refill makes them hold theta0 again
  bool any_inplace = false;
  bool any_inplace_rel = false;
  bool theta0_resident = true;
  DevTensor* d_tensors = nullptr;
  Chunk* d_chunks = nullptr;
  DevScalars* d_scal = nullptr;
  StatPartial* d_partials = nullptr;
  GradPtr* d_grads = nullptr;
  RoundKeys keys;
  int sm_count = 1;
  int64_t chunk_elems = kMaxChunkElems;  // work-chunk size of this list
  int32_t active = 0;
  int64_t scalars_step = -1;  // step whose scalars the table holds
  int64_t sim_step = -1;      // step of the last forward: the only step whose mask a gradient map may regenerate
  bool scalars_sigma = false; // the table's sigma_t are current
  std::vector<GradPtr> h_grads;
  bool grads_uploaded = false;
  // the fused AdamW table lives in the same workspace region as the gradient
  // table: uploading one invalidates the other
  std::vector<AdamPtr> h_adams;
  bool adams_uploaded = false;
  // work-list forward launch (with the statistics of sigma_rel tensors)
  bool fused = false;
  bool wide = false;  // the bf16 fused launch carries statistics items: its four-CTA build
  std::vector<int32_t> h_items;
  int32_t item_begin[kMaxRanges] = {0, 0};
  int32_t item_count[kMaxRanges] = {0, 0};
  int32_t* d_items = nullptr;
  int32_t* d_sync = nullptr;  // see sync_words()
  uint32_t epoch = 0;
  // optional per-kernel timing
  bool timing = false;
  struct Mark { int kind; cudaEvent_t start, stop; };
  std::vector<Mark> marks;
  std::vector<cudaEvent_t> event_pool;
  double ms[4] = {0, 0, 0, 0};
  int64_t launches[4] = {0, 0, 0, 0};
  ~smat_ctx() {
    for (auto& m : marks) { event_pool.push_back(m.start); event_pool.push_back(m.stop); }
    for (cudaEvent_t e : event_pool) cudaEventDestroy(e);
  }
};

namespace {

cudaEvent_t take_event(smat_ctx* c) {
  if (!c->event_pool.empty()) {
    cudaEvent_t e = c->event_pool.back();
    c->event_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

// Bracket one launch with events on its stream when timing is enabled.
struct Timed {
  smat_ctx* c;
  int kind;
  cudaStream_t s;
  cudaEvent_t start = nullptr;
  Timed(smat_ctx* c_, int kind_, cudaStream_t s_) : c(c_), kind(kind_), s(s_) {
    if (c->timing && (start = take_event(c)) != nullptr) cudaEventRecord(start, s);
  }
  void done() {
    if (!start) return;
    cudaEvent_t stop = take_event(c);
    if (!stop) { c->event_pool.push_back(start); return; }
    cudaEventRecord(stop, s);
    c->marks.push_back({kind, start, stop});
  }
};

KArgs base_args(const smat_ctx* c, uint32_t step) {
  KArgs a;
  std::memset(&a, 0, sizeof(a));
  a.tensors = c->d_tensors;
  a.chunks = c->d_chunks;
  a.scal = c->d_scal;
  a.partials = c->d_partials;
  a.grads = c->d_grads;
  a.adams = reinterpret_cast<const AdamPtr*>(c->d_grads);
  a.key = c->keys;
  a.step = step;
  a.n_tensors = (int32_t)c->desc.size();
  a.alpha_min = c->cfg.alpha_min;
  a.alpha_width = c->cfg.alpha_max - c->cfg.alpha_min;
  a.alpha_mode = c->cfg.alpha_mode;
  a.grad_unit = std::min(c->chunk_elems, kMaxGradUnitElems);
  a.grad_units = (int32_t)(c->chunk_elems / a.grad_unit);
  if (c->d_sync) {
    a.work_counter = c->d_sync;
    a.error = c->d_sync + 2;
    a.tensor_done = c->d_sync + 4;
    a.ready = reinterpret_cast<uint32_t*>(c->d_sync + 4 + c->desc.size());
  }
  return a;
}

// Work list of the fused launch for one dtype range: statistics items (chunk
// c at key 2c) and forward items; a forward item of a sigma_rel tensor gets
// key 2 (last + lead + its position in the tensor) + 1, so all statistics
// items of its tensor come first and the forward trails by `lead` chunks.
void build_items(smat_ctx* c, int dt, int64_t lead) {
  std::vector<std::pair<int64_t, int32_t>> keyed;
  for (int64_t ci = c->range_begin[dt]; ci < c->range_end[dt]; ++ci) {
    const Chunk& ch = c->h_chunks[(size_t)ci];
    const DevTensor& T = c->h_tensors[ch.tensor];
    const int64_t first = T.chunk_first, last = T.chunk_first + T.n_chunks - 1;
    if (T.flags & TF_SIGMA_REL) {
      keyed.push_back({2 * ci, (int32_t)ci});
      keyed.push_back({2 * (last + lead + (ci - first)) + 1, (int32_t)(ci | (int64_t)kItemForward)});
    } else {
      keyed.push_back({2 * ci + 1, (int32_t)(ci | (int64_t)kItemForward)});
    }
  }
  std::stable_sort(keyed.begin(), keyed.end(),
                   [](const std::pair<int64_t, int32_t>& x, const std::pair<int64_t, int32_t>& y) { return x.first < y.first; });
  c->item_begin[dt] = (int32_t)c->h_items.size();
  for (auto& kv : keyed) c->h_items.push_back(kv.second);
  c->item_count[dt] = (int32_t)keyed.size();
}

int grid_for(const smat_ctx* c, int64_t chunks, int dtype) {
  const int64_t resident = (int64_t)c->sm_count *
                           streaming_ctas_per_sm(dtype, c->cfg.noise, c->cfg.alpha_mode == SMAT_ALPHA_PER_ELEMENT, c->rounds);
  return (int)(chunks < resident ? chunks : resident);
}

// Rows a2 + a1: delta statistics (if needed) then the per-call scalars.
smat_status run_scalars(smat_ctx* c, uint32_t step, bool with_sigma, cudaStream_t s) {
  KArgs a = base_args(c, step);
  cudaError_t e;
  const bool stats = with_sigma && c->any_sigma_rel;
  if (stats) {
    for (int dt = 0; dt < 2; ++dt) {
      a.chunk_begin = c->range_begin[dt];
      a.chunk_end = c->range_end[dt];
      if (a.chunk_end <= a.chunk_begin) continue;
      Timed t(c, 0, s);
      e = launch_delta_stats(a, grid_for(c, a.chunk_end - a.chunk_begin, dt), dt, s);
      t.done();
      if (e != cudaSuccess) return cuda_fail(e, "delta statistics launch");
    }
  }
  a.chunk_begin = 0;
  a.chunk_end = 0;
  a.with_sigma = stats ? 1 : 0;
  if (a.n_tensors == 0) return SMAT_OK;
  Timed t(c, 1, s);
  e = launch_scalars(a, c->cfg.noise, c->rounds, s);
  t.done();
  if (e != cudaSuccess) return cuda_fail(e, "scalars launch");
  c->scalars_step = step;
  c->scalars_sigma = with_sigma;
  return SMAT_OK;
}

}  // namespace

extern "C" {

size_t smat_workspace_bytes(const smat_tensor_desc* tensors, int32_t n_tensors, const smat_config* cfg) {
  if (check_config(cfg) != SMAT_OK) return 0;
  int64_t nc = 0;
  bool rel = false;
  int64_t cs = 0;
  if (check_tensors(tensors, n_tensors, cfg, &nc, &rel, &cs) != SMAT_OK) return 0;
  return layout_for(n_tensors, nc, rel).total;
}

smat_status smat_init(smat_ctx** out, const smat_tensor_desc* tensors, int32_t n_tensors,
                      const smat_config* cfg, void* d_workspace, size_t workspace_bytes,
                      smat_stream_t stream) {
  if (!out) return fail(SMAT_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  smat_status st = check_config(cfg);
  if (st != SMAT_OK) return st;
  int64_t nc = 0;
  bool rel = false;
  int64_t cs = 0;
  st = check_tensors(tensors, n_tensors, cfg, &nc, &rel, &cs);
  if (st != SMAT_OK) return st;
  const Layout L = layout_for(n_tensors, nc, rel);
  if (!d_workspace) return fail(SMAT_ERR_WORKSPACE, "workspace is NULL");
  if ((uintptr_t)d_workspace % kAlign) return fail(SMAT_ERR_WORKSPACE, "workspace not 256-byte aligned");
  if (workspace_bytes < L.total)
    return fail(SMAT_ERR_WORKSPACE, "workspace %zu bytes < %zu needed", workspace_bytes, L.total);
  st = check_gpu_access(tensors, n_tensors);
  if (st != SMAT_OK) return st;

  smat_ctx* c = new smat_ctx();
  c->desc.assign(tensors, tensors + n_tensors);
  c->cfg = *cfg;
  c->rounds = (cfg->philox_rounds == 7 ? 7 : 10) | (cfg->draw_bits == 16 ? kDraw16 : 0);
  const bool d16 = cfg->draw_bits == 16;
  c->any_sigma_rel = rel;
  c->chunk_elems = cs;
  c->keys = make_keys(cfg->seed);
  char* ws = static_cast<char*>(d_workspace);
  c->d_tensors = reinterpret_cast<DevTensor*>(ws + L.tensors);
  c->d_chunks = reinterpret_cast<Chunk*>(ws + L.chunks);
  c->d_scal = reinterpret_cast<DevScalars*>(ws + L.scal);
  c->d_partials = rel ? reinterpret_cast<StatPartial*>(ws + L.partials) : nullptr;
  c->d_grads = reinterpret_cast<GradPtr*>(ws + L.grads);
  c->d_items = reinterpret_cast<int32_t*>(ws + L.items);
  c->d_sync = reinterpret_cast<int32_t*>(ws + L.sync);
  c->fused = !(cfg->flags & SMAT_FLAG_UNFUSED_STATS);

  c->h_tensors.resize(n_tensors);
  c->h_chunks.reserve((size_t)nc);
  for (int dt = 0; dt < 2; ++dt) {
    c->range_begin[dt] = (int64_t)c->h_chunks.size();
    for (int32_t k = 0; k < n_tensors; ++k) {
      const smat_tensor_desc& d = tensors[k];
      if (d.dtype != dt) continue;
      DevTensor& T = c->h_tensors[k];
      std::memset(&T, 0, sizeof(T));
      T.theta = d.theta;
      T.theta0 = d.theta0;
      T.sim = d.sim;
      T.numel = d.numel;
      T.elem_offset = d.elem_offset;
      T.tid = d.tensor_id;
      T.dtype = d.dtype;
      T.sigma = d.sigma;
      T.sigma_rel = d.sigma_rel;
      // Eq. smat-mask: keep with probability p_keep = 1 - p, rescale by 1 / p_keep.
      // The threshold is on a 32-bit draw (its high byte, then on a tie the low
      // 24 bits), or on a 16-bit draw with the 16-bit option (t_hi holds it;
      // t_lo = 0, so there are no ties).
      const int draw = d16 ? 16 : 32;
      const uint64_t thr = (uint64_t)std::floor((double)d.keep_prob * (double)(uint64_t(1) << draw));
      T.inv_keep = d.keep_prob > 0.0f ? (float)(1.0 / (double)d.keep_prob) : 0.0f;
      uint32_t flags = 0;
      if (thr < (uint64_t(1) << draw)) {
        flags |= TF_MASK;
        T.t_hi = d16 ? (uint32_t)thr : (uint32_t)(thr >> 24);
        T.t_lo = d16 ? 0u : (uint32_t)(thr & 0xFFFFFFu);
      }
      // 256-bit vector accesses need 32-byte aligned addresses; groups of 16
      // elements start at multiples of 16 elements from the base pointer.
      if (((uintptr_t)d.theta % 32 == 0) && ((uintptr_t)d.theta0 % 32 == 0) &&
          ((uintptr_t)d.sim % 32 == 0) && (d.elem_offset % 16 == 0))
        flags |= TF_VEC;
      if (d.sigma_rel > 0.0f) flags |= TF_SIGMA_REL;
      if (d.numel > 0 && d.sim == d.theta0) {
        flags |= TF_INPLACE;
        c->any_inplace = true;
        c->any_inplace_rel = c->any_inplace_rel || d.sigma_rel > 0.0f;
      }
      T.flags = flags;
      T.chunk_first = (int32_t)c->h_chunks.size();
      const int64_t m = chunks_of(d.numel, cs);
      T.n_chunks = (int32_t)m;
      for (int64_t j = 0; j < m; ++j) {
        Chunk ch;
        ch.tensor = k;
        ch.pad = 0;
        ch.begin = j * cs;
        ch.end = (j + 1) * cs < d.numel ? (j + 1) * cs : d.numel;
        c->h_chunks.push_back(ch);
      }
    }
    c->range_end[dt] = (int64_t)c->h_chunks.size();
  }

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&c->sm_count, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess && n_tensors > 0)
    e = cudaMemcpyAsync(c->d_tensors, c->h_tensors.data(), sizeof(DevTensor) * (size_t)n_tensors,
                        cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess && nc > 0)
    e = cudaMemcpyAsync(c->d_chunks, c->h_chunks.data(), sizeof(Chunk) * (size_t)nc,
                        cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->d_sync, 0, sizeof(int32_t) * sync_words(n_tensors), stream);
  c->wide = rel && cfg->alpha_mode != SMAT_ALPHA_PER_ELEMENT && cfg->noise != SMAT_NOISE_LAPLACE && !c->any_inplace;
  if (e == cudaSuccess && c->fused) {
    // lead of about one grid width of the bf16 forward (one, two and four
    // measured on the 7B list: one is fastest)
    const int64_t lead = (int64_t)c->sm_count *
                         (c->wide ? fused_wide_occ(cfg->noise, c->rounds)
                                  : streaming_ctas_per_sm(SMAT_BF16, cfg->noise,
                                                          cfg->alpha_mode == SMAT_ALPHA_PER_ELEMENT, c->rounds));
    for (int dt = 0; dt < 2; ++dt) build_items(c, dt, lead);
    if (!c->h_items.empty())
      e = cudaMemcpyAsync(c->d_items, c->h_items.data(), sizeof(int32_t) * c->h_items.size(),
                          cudaMemcpyHostToDevice, stream);
  }
  // The host vectors are pageable: the copies above have been staged when
  // they return, but keep the data in the context anyway for its lifetime.
  if (e != cudaSuccess) {
    delete c;
    return cuda_fail(e, "smat_init upload");
  }
  *out = c;
  return SMAT_OK;
}

smat_status smat_simulate_multi(smat_ctx* c, uint32_t step, smat_stream_t stream) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  if (c->active != 0)
    return fail(SMAT_ERR_STATE, "simulate called while the simulated storage is active; swap back first");
  if (c->any_inplace && !c->theta0_resident)
    return fail(SMAT_ERR_STATE, "in-place tensors: theta0 has not been refilled since the last forward");
  c->theta0_resident = false;  // the forward below overwrites it
  c->sim_step = -1;            // set again once every launch of this forward is enqueued
  if (c->fused) {
    // a1 (alpha, c; sigma of fixed-sigma tensors; counter reset), then a3 (with a2
    // for sigma_rel tensors) in one work-list launch
    smat_status st = run_scalars(c, step, false, stream);
    if (st != SMAT_OK) return st;
    c->scalars_sigma = true;
    c->epoch += 1;
    if (c->epoch == 0) c->epoch = 1;
    KArgs a = base_args(c, step);
    a.epoch = c->epoch;
    for (int dt = 0; dt < 2; ++dt) {
      if (c->item_count[dt] == 0) continue;
      a.items = c->d_items + c->item_begin[dt];
      a.n_items = c->item_count[dt];
      a.work_counter = c->d_sync + dt;
      const bool wide = c->wide && dt == SMAT_BF16;
      int grid = grid_for(c, c->range_end[dt] - c->range_begin[dt], dt);
      if (wide) {
        const int64_t chunks = c->range_end[dt] - c->range_begin[dt];
        const int64_t resident = (int64_t)c->sm_count * fused_wide_occ(c->cfg.noise, c->rounds);
        grid = (int)(chunks < resident ? chunks : resident);
      }
      Timed t(c, 2, stream);
      const cudaError_t e = launch_stats_simulate(a, grid, dt, c->cfg.noise, c->cfg.alpha_mode == SMAT_ALPHA_PER_ELEMENT,
                                                  c->rounds, c->any_inplace, wide, stream);
      t.done();
      if (e != cudaSuccess) return cuda_fail(e, "fused statistics + forward launch");
    }
    c->sim_step = step;
    return SMAT_OK;
  }
  smat_status st = run_scalars(c, step, true, stream);
  if (st != SMAT_OK) return st;
  KArgs a = base_args(c, step);
  for (int dt = 0; dt < 2; ++dt) {
    a.chunk_begin = c->range_begin[dt];
    a.chunk_end = c->range_end[dt];
    if (a.chunk_end <= a.chunk_begin) continue;
    Timed t(c, 2, stream);
    const cudaError_t e = launch_simulate(a, grid_for(c, a.chunk_end - a.chunk_begin, dt), dt, c->cfg.noise,
                                          c->cfg.alpha_mode == SMAT_ALPHA_PER_ELEMENT, c->rounds, c->any_inplace,
                                          stream);
    t.done();
    if (e != cudaSuccess) return cuda_fail(e, "simulate launch");
  }
  c->sim_step = step;
  return SMAT_OK;
}

smat_status smat_grad_map_multi(smat_ctx* c, uint32_t step, const void* const* g_sim, void* const* g_out,
                                int32_t gdtype, int32_t accumulate, smat_stream_t stream) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  if (gdtype != SMAT_F32 && gdtype != SMAT_BF16)
    return fail(SMAT_ERR_UNSUPPORTED, "gradient dtype %d not supported", gdtype);
  // Eq. smat-gradient maps g~ through the mask of the forward that produced
  // theta~ (regenerated, App. D): only the step of the last forward qualifies.
  if (c->sim_step != (int64_t)step) {
    if (c->sim_step < 0)
      return fail(SMAT_ERR_STATE, "gradient map for step %u, but no forward has run on this context", step);
    return fail(SMAT_ERR_STATE, "gradient map for step %u, but the last forward on this context was step %lld", step,
                (long long)c->sim_step);
  }
  const int32_t n = (int32_t)c->desc.size();
  if (n > 0 && (!g_sim || !g_out)) return fail(SMAT_ERR_INVALID_ARG, "gradient pointer arrays are NULL");
  const size_t es = elem_size(gdtype);
  std::vector<GradPtr> g((size_t)n);
  for (int32_t k = 0; k < n; ++k) {
    const smat_tensor_desc& d = c->desc[k];
    GradPtr& p = g[k];
    std::memset(&p, 0, sizeof(p));
    p.g_sim = g_sim[k];
    p.g_out = g_out[k];
    if (d.numel > 0) {
      if (!p.g_sim || !p.g_out) return fail(SMAT_ERR_INVALID_ARG, "tensor %d: NULL gradient pointer", k);
      if ((uintptr_t)p.g_sim % es || (uintptr_t)p.g_out % es)
        return fail(SMAT_ERR_ALIGNMENT, "tensor %d: gradient pointer not aligned to %zu bytes", k, es);
      const size_t bytes = es * (size_t)d.numel;
      if (p.g_sim != p.g_out && overlaps(p.g_sim, bytes, p.g_out, bytes))
        return fail(SMAT_ERR_INVALID_ARG, "tensor %d: g_out partially overlaps g_sim", k);
    }
    p.vec = ((uintptr_t)p.g_sim % 32 == 0 && (uintptr_t)p.g_out % 32 == 0 && d.elem_offset % 16 == 0) ? 1u : 0u;
  }
  if (!c->grads_uploaded || g.size() != c->h_grads.size() ||
      (n > 0 && std::memcmp(g.data(), c->h_grads.data(), sizeof(GradPtr) * (size_t)n) != 0)) {
    c->h_grads.swap(g);
    if (n > 0) {
      const cudaError_t e = cudaMemcpyAsync(c->d_grads, c->h_grads.data(), sizeof(GradPtr) * (size_t)n,
                                            cudaMemcpyHostToDevice, stream);
      if (e != cudaSuccess) return cuda_fail(e, "gradient table upload");
    }
    c->grads_uploaded = true;
    c->adams_uploaded = false;
  }
  if (c->scalars_step != (int64_t)step) {
    const smat_status st = run_scalars(c, step, false, stream);
    if (st != SMAT_OK) return st;
  }
  KArgs a = base_args(c, step);
  a.chunk_begin = 0;
  a.chunk_end = (int64_t)c->h_chunks.size();
  const int64_t resident = (int64_t)c->sm_count *
                           grad_map_occ(gdtype, c->cfg.alpha_mode == SMAT_ALPHA_PER_ELEMENT, accumulate != 0, c->rounds);
  const int grid = (int)(a.chunk_end < resident ? a.chunk_end : resident);
  if (a.chunk_end <= 0) return SMAT_OK;
  Timed t(c, 3, stream);
  const cudaError_t e = launch_grad_map(a, grid, gdtype, c->cfg.alpha_mode == SMAT_ALPHA_PER_ELEMENT,
                                       accumulate != 0, c->rounds, stream);
  t.done();
  if (e != cudaSuccess) return cuda_fail(e, "gradient map launch");
  return SMAT_OK;
}

smat_status smat_grad_map_adamw_multi(smat_ctx* c, uint32_t step, const void* const* g_sim, float* const* m1,
                                      float* const* m2, int32_t gdtype, const smat_adamw* opt,
                                      smat_stream_t stream) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  if (!opt) return fail(SMAT_ERR_INVALID_ARG, "opt is NULL");
  if (gdtype != SMAT_F32 && gdtype != SMAT_BF16)
    return fail(SMAT_ERR_UNSUPPORTED, "gradient dtype %d not supported", gdtype);
  if (!(std::isfinite(opt->lr) && opt->lr >= 0.0f))
    return fail(SMAT_ERR_INVALID_ARG, "lr must be finite and >= 0");
  if (!(opt->beta1 >= 0.0f && opt->beta1 < 1.0f) || !(opt->beta2 >= 0.0f && opt->beta2 < 1.0f))
    return fail(SMAT_ERR_INVALID_ARG, "beta1 and beta2 must lie in [0, 1)");
  if (!(std::isfinite(opt->eps) && opt->eps > 0.0f)) return fail(SMAT_ERR_INVALID_ARG, "eps must be finite and > 0");
  if (!(std::isfinite(opt->weight_decay) && opt->weight_decay >= 0.0f))
    return fail(SMAT_ERR_INVALID_ARG, "weight_decay must be finite and >= 0");
  if (opt->step < 1) return fail(SMAT_ERR_INVALID_ARG, "optimizer step %d: must be >= 1", opt->step);
  // same rule as the gradient map: the mask of the forward that produced the
  // gradient's theta~ (App. D)
  if (c->sim_step != (int64_t)step) {
    if (c->sim_step < 0)
      return fail(SMAT_ERR_STATE, "gradient map for step %u, but no forward has run on this context", step);
    return fail(SMAT_ERR_STATE, "gradient map for step %u, but the last forward on this context was step %lld", step,
                (long long)c->sim_step);
  }
  // the update writes theta, so the original storage must be the one the
  // model reads (Sec. 4.3: the storage is switched back before the update)
  if (c->active != 0) return fail(SMAT_ERR_STATE, "the simulated storage is active: switch back before the update");
  const int32_t n = (int32_t)c->desc.size();
  if (n > 0 && (!g_sim || !m1 || !m2)) return fail(SMAT_ERR_INVALID_ARG, "pointer arrays are NULL");
  const size_t es = elem_size(gdtype);
  std::vector<AdamPtr> t((size_t)n);
  for (int32_t k = 0; k < n; ++k) {
    const smat_tensor_desc& d = c->desc[k];
    AdamPtr& p = t[k];
    std::memset(&p, 0, sizeof(p));
    p.g_sim = g_sim[k];
    p.m1 = m1[k];
    p.m2 = m2[k];
    if (d.numel > 0) {
      if (!p.g_sim || !p.m1 || !p.m2) return fail(SMAT_ERR_INVALID_ARG, "tensor %d: NULL pointer", k);
      if ((uintptr_t)p.g_sim % es) return fail(SMAT_ERR_ALIGNMENT, "tensor %d: g_sim not aligned to %zu bytes", k, es);
      if ((uintptr_t)p.m1 % 4 || (uintptr_t)p.m2 % 4)
        return fail(SMAT_ERR_ALIGNMENT, "tensor %d: moment buffers not 4-byte aligned", k);
      const size_t gb = es * (size_t)d.numel, mb = 4 * (size_t)d.numel;
      const size_t tb = elem_size(d.dtype) * (size_t)d.numel;
      if (overlaps(p.m1, mb, p.m2, mb) || overlaps(p.m1, mb, d.theta, tb) || overlaps(p.m2, mb, d.theta, tb) ||
          overlaps(p.g_sim, gb, d.theta, tb) || overlaps(p.g_sim, gb, p.m1, mb) || overlaps(p.g_sim, gb, p.m2, mb))
        return fail(SMAT_ERR_INVALID_ARG, "tensor %d: theta, g_sim, m1 and m2 must not overlap", k);
    }
    p.vec = ((uintptr_t)p.g_sim % 32 == 0 && (uintptr_t)p.m1 % 32 == 0 && (uintptr_t)p.m2 % 32 == 0 &&
             (uintptr_t)d.theta % 32 == 0 && d.elem_offset % 16 == 0)
                ? 1u
                : 0u;
  }
  if (!c->adams_uploaded || t.size() != c->h_adams.size() ||
      (n > 0 && std::memcmp(t.data(), c->h_adams.data(), sizeof(AdamPtr) * (size_t)n) != 0)) {
    c->h_adams.swap(t);
    if (n > 0) {
      const cudaError_t e = cudaMemcpyAsync(c->d_grads, c->h_adams.data(), sizeof(AdamPtr) * (size_t)n,
                                            cudaMemcpyHostToDevice, stream);
      if (e != cudaSuccess) return cuda_fail(e, "optimizer table upload");
    }
    c->adams_uploaded = true;
    c->grads_uploaded = false;
  }
  if (c->scalars_step != (int64_t)step) {
    const smat_status st = run_scalars(c, step, false, stream);
    if (st != SMAT_OK) return st;
  }
  KArgs a = base_args(c, step);
  const double b1 = opt->beta1, b2 = opt->beta2, tt = (double)opt->step;
  a.adam.decay = (float)(1.0 - (double)opt->lr * (double)opt->weight_decay);
  a.adam.b1 = opt->beta1;
  a.adam.omb1 = (float)(1.0 - b1);
  a.adam.b2 = opt->beta2;
  a.adam.omb2 = (float)(1.0 - b2);
  a.adam.bc2 = (float)std::sqrt(1.0 - std::pow(b2, tt));
  a.adam.step = (float)((double)opt->lr / (1.0 - std::pow(b1, tt)));
  a.adam.eps = opt->eps;
  a.chunk_begin = 0;
  a.chunk_end = (int64_t)c->h_chunks.size();
  if (a.chunk_end <= 0) return SMAT_OK;
  // one launch per parameter dtype (the kernel is specialised on it)
  const bool pe = c->cfg.alpha_mode == SMAT_ALPHA_PER_ELEMENT;
  for (int dt = 0; dt < 2; ++dt) {
    a.chunk_begin = c->range_begin[dt];
    a.chunk_end = c->range_end[dt];
    if (a.chunk_end <= a.chunk_begin) continue;
    const int pdt = dt == 0 ? SMAT_F32 : SMAT_BF16;
    const int64_t units = (a.chunk_end - a.chunk_begin) * (int64_t)a.grad_units;
    const int64_t resident = (int64_t)c->sm_count * grad_map_adamw_occ(gdtype, pdt, pe, c->rounds);
    const int grid = (int)(units < resident ? units : resident);
    Timed tm(c, 3, stream);
    const cudaError_t e = launch_grad_map_adamw(a, grid, gdtype, pdt, pe, c->rounds, stream);
    tm.done();
    if (e != cudaSuccess) return cuda_fail(e, "fused AdamW launch");
  }
  return SMAT_OK;
}

smat_status smat_swap(smat_ctx* c, int32_t* active_out) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  c->active ^= 1;
  if (active_out) *active_out = c->active;
  return SMAT_OK;
}

smat_status smat_refill_theta0(smat_ctx* c, const void* const* h_theta0, smat_stream_t stream) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  if (c->active != 0)
    return fail(SMAT_ERR_STATE, "refill while the simulated storage is active: the model reads those buffers");
  const int32_t n = (int32_t)c->desc.size();
  if (c->any_inplace && !h_theta0) return fail(SMAT_ERR_INVALID_ARG, "h_theta0 is NULL");
  for (int32_t k = 0; k < n; ++k) {
    if (!(c->h_tensors[(size_t)k].flags & TF_INPLACE)) continue;
    if (!h_theta0[k]) return fail(SMAT_ERR_INVALID_ARG, "tensor %d: h_theta0 entry is NULL", k);
  }
  for (int32_t k = 0; k < n; ++k) {
    const smat_tensor_desc& d = c->desc[(size_t)k];
    if (!(c->h_tensors[(size_t)k].flags & TF_INPLACE)) continue;
    const cudaError_t e = cudaMemcpyAsync(d.sim, h_theta0[k], elem_size(d.dtype) * (size_t)d.numel,
                                          cudaMemcpyHostToDevice, stream);
    if (e != cudaSuccess) return cuda_fail(e, "theta0 refill copy");
  }
  c->theta0_resident = true;
  return SMAT_OK;
}

smat_status smat_mark_theta0_resident(smat_ctx* c) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  if (c->active != 0)
    return fail(SMAT_ERR_STATE, "the simulated storage is active: its buffers hold theta~");
  c->theta0_resident = true;
  return SMAT_OK;
}

smat_status smat_active(const smat_ctx* c, int32_t* active_out) {
  if (!c || !active_out) return fail(SMAT_ERR_INVALID_ARG, "NULL argument");
  *active_out = c->active;
  return SMAT_OK;
}

smat_status smat_mask_bits(smat_ctx* c, uint32_t step, int32_t tensor_index, uint32_t* d_bits,
                           smat_stream_t stream) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  if (tensor_index < 0 || tensor_index >= (int32_t)c->desc.size())
    return fail(SMAT_ERR_INVALID_ARG, "tensor_index %d out of range", tensor_index);
  const int64_t numel = c->desc[tensor_index].numel;
  if (numel == 0) return SMAT_OK;
  if (!d_bits) return fail(SMAT_ERR_INVALID_ARG, "d_bits is NULL");
  if ((uintptr_t)d_bits % 4) return fail(SMAT_ERR_ALIGNMENT, "d_bits not 4-byte aligned");
  KArgs a = base_args(c, step);
  a.bits = d_bits;
  a.tensor_index = tensor_index;
  const cudaError_t e = launch_mask_bits(a, numel, c->rounds, stream);
  if (e != cudaSuccess) return cuda_fail(e, "mask bits launch");
  return SMAT_OK;
}

smat_status smat_tensor_scalars(smat_ctx* c, uint32_t step, float* d_out, smat_stream_t stream) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  const size_t n = c->desc.size();
  if (n == 0) return SMAT_OK;
  if (!d_out) return fail(SMAT_ERR_INVALID_ARG, "d_out is NULL");
  if ((uintptr_t)d_out % 4) return fail(SMAT_ERR_ALIGNMENT, "d_out not 4-byte aligned");
  if (c->any_inplace_rel && !c->theta0_resident)
    return fail(SMAT_ERR_STATE, "in-place sigma_rel tensors: theta0 is not resident (refill it first)");
  const smat_status st = run_scalars(c, step, true, stream);
  if (st != SMAT_OK) return st;
  const cudaError_t e = cudaMemcpyAsync(d_out, c->d_scal, sizeof(DevScalars) * n, cudaMemcpyDeviceToDevice, stream);
  if (e != cudaSuccess) return cuda_fail(e, "scalars copy");
  return SMAT_OK;
}

smat_status smat_debug_fused(smat_ctx* c, uint32_t step, const int32_t* d_items, int32_t n_items,
                             uint32_t epoch_skew, smat_stream_t stream) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  if (!c->any_sigma_rel) return fail(SMAT_ERR_STATE, "context has no sigma_rel tensor");
  if (c->any_inplace) return fail(SMAT_ERR_STATE, "test hook not available with in-place tensors");
  if (n_items < 0 || (n_items > 0 && !d_items)) return fail(SMAT_ERR_INVALID_ARG, "bad item list");
  if (c->range_end[SMAT_BF16] <= c->range_begin[SMAT_BF16]) return fail(SMAT_ERR_STATE, "no bf16 tensors");
  // items must name chunks of the bf16 range; checked on the host copy the caller passes through
  std::vector<int32_t> h((size_t)n_items);
  cudaError_t e = n_items ? cudaMemcpyAsync(h.data(), d_items, sizeof(int32_t) * (size_t)n_items,
                                            cudaMemcpyDeviceToHost, stream) : cudaSuccess;
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cuda_fail(e, "item list read");
  for (int32_t v : h) {
    const int64_t ci = (int64_t)((uint32_t)v & ~kItemForward);
    if (ci < c->range_begin[SMAT_BF16] || ci >= c->range_end[SMAT_BF16])
      return fail(SMAT_ERR_INVALID_ARG, "item names chunk %lld outside the bf16 range", (long long)ci);
  }
  smat_status st = run_scalars(c, step, false, stream);
  if (st != SMAT_OK) return st;
  c->epoch += 1;
  if (c->epoch == 0) c->epoch = 1;
  KArgs a = base_args(c, step);
  a.epoch = c->epoch + epoch_skew;
  a.items = d_items;
  a.n_items = n_items;
  a.work_counter = c->d_sync + SMAT_BF16;
  e = launch_stats_simulate_bf16(a, grid_for(c, c->range_end[SMAT_BF16] - c->range_begin[SMAT_BF16], SMAT_BF16),
                                 c->cfg.noise, c->cfg.alpha_mode == SMAT_ALPHA_PER_ELEMENT, c->rounds, false, stream);
  if (e != cudaSuccess) return cuda_fail(e, "fused launch");
  c->scalars_step = -1;  // sigma_t of this call may be incomplete
  c->sim_step = -1;      // and its forward too
  return SMAT_OK;
}

smat_status smat_poll_errors(smat_ctx* c, smat_stream_t stream, int32_t* errors_out) {
  if (!c || !errors_out) return fail(SMAT_ERR_INVALID_ARG, "NULL argument");
  int32_t v = 0;
  cudaError_t e = cudaMemcpyAsync(&v, c->d_sync + 2, sizeof(int32_t), cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e == cudaSuccess && v != 0) e = cudaMemsetAsync(c->d_sync + 2, 0, sizeof(int32_t), stream);
  if (e != cudaSuccess) return cuda_fail(e, "error flag read");
  *errors_out = v;
  return SMAT_OK;
}

smat_status smat_timing_enable(smat_ctx* c, int32_t enable) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  for (auto& m : c->marks) {
    c->event_pool.push_back(m.start);
    c->event_pool.push_back(m.stop);
  }
  c->marks.clear();
  for (int k = 0; k < 4; ++k) {
    c->ms[k] = 0.0;
    c->launches[k] = 0;
  }
  c->timing = enable != 0;
  return SMAT_OK;
}

smat_status smat_timing_read(smat_ctx* c, double* ms_out, int64_t* launches_out) {
  if (!c) return fail(SMAT_ERR_INVALID_ARG, "ctx is NULL");
  for (auto& m : c->marks) {
    cudaError_t e = cudaEventSynchronize(m.stop);
    float ms = 0.0f;
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, m.start, m.stop);
    if (e != cudaSuccess) return cuda_fail(e, "timing event");
    c->ms[m.kind] += ms;
    c->launches[m.kind] += 1;
    c->event_pool.push_back(m.start);
    c->event_pool.push_back(m.stop);
  }
  c->marks.clear();
  for (int k = 0; k < 4; ++k) {
    if (ms_out) ms_out[k] = c->ms[k];
    if (launches_out) launches_out[k] = c->launches[k];
  }
  return SMAT_OK;
}

smat_status smat_destroy(smat_ctx* c) {
  delete c;
  return SMAT_OK;
}

smat_status smat_debug_philox(const uint32_t* d_ctr, int64_t n, uint64_t seed, int32_t rounds,
                              uint32_t* d_out, uint32_t* d_out_ref, smat_stream_t stream) {
  if (n < 0) return fail(SMAT_ERR_INVALID_ARG, "n < 0");
  if (n == 0) return SMAT_OK;
  if (!d_ctr || !d_out) return fail(SMAT_ERR_INVALID_ARG, "NULL pointer");
  if (rounds != 7 && rounds != 10) return fail(SMAT_ERR_UNSUPPORTED, "rounds %d not supported", rounds);
  if (d_out_ref && rounds != 10) return fail(SMAT_ERR_UNSUPPORTED, "cuRAND reference needs 10 rounds");
  const cudaError_t e = launch_debug_philox(d_ctr, n, make_keys(seed), rounds, d_out, d_out_ref, stream);
  if (e != cudaSuccess) return cuda_fail(e, "philox launch");
  return SMAT_OK;
}

smat_status smat_debug_noise_unit(const uint32_t* d_words, int64_t n, int32_t noise, float* d_out,
                                  smat_stream_t stream) {
  if (n < 0) return fail(SMAT_ERR_INVALID_ARG, "n < 0");
  if (n == 0) return SMAT_OK;
  if (!d_words || !d_out) return fail(SMAT_ERR_INVALID_ARG, "NULL pointer");
  if (noise != SMAT_NOISE_UNIFORM && noise != SMAT_NOISE_GAUSSIAN && noise != SMAT_NOISE_LAPLACE)
    return fail(SMAT_ERR_UNSUPPORTED, "noise %d not supported", noise);
  const cudaError_t e = launch_debug_noise_unit(d_words, n, noise, d_out, stream);
  if (e != cudaSuccess) return cuda_fail(e, "noise transform launch");
  return SMAT_OK;
}

const char* smat_status_string(smat_status s) {
  switch (s) {
    case SMAT_OK: return "SMAT_OK";
    case SMAT_ERR_INVALID_ARG: return "SMAT_ERR_INVALID_ARG";
    case SMAT_ERR_UNSUPPORTED: return "SMAT_ERR_UNSUPPORTED";
    case SMAT_ERR_ALIGNMENT: return "SMAT_ERR_ALIGNMENT";
    case SMAT_ERR_WORKSPACE: return "SMAT_ERR_WORKSPACE";
    case SMAT_ERR_STATE: return "SMAT_ERR_STATE";
    case SMAT_ERR_CUDA: return "SMAT_ERR_CUDA";
  }
  return "SMAT_ERR_UNKNOWN";
}

const char* smat_last_error(void) { return g_last_error.c_str(); }

int32_t smat_abi_version(void) { return SMAT_ABI_VERSION; }

}  // extern "C"
