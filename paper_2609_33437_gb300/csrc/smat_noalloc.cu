// smat_delta_sigma_noalloc: the delta-statistics computation of one tensor
// (sigma = sigma_rel * population std of theta - theta0) without any device
// allocation, for callers that cannot allocate device memory: for example a
// plugin inside a host framework that owns all of the GPU's memory, or code
// that must not grow a memory pool once a job is running. Its per-chunk
// partial sums live in a fixed file-scope device array instead of a
// caller-provided workspace.
//
// The array holds kNoAllocMaxChunks partials (256 KiB), one per 2^16-element
// chunk; every GPU that loads this library keeps it for the life of the
// process. Tensors of more than kNoAllocMaxChunks * 2^16 elements are rejected.

#include <mutex>

#include "smat_device.cuh"
#include "smat.h"

namespace smat {
namespace {

constexpr int64_t kNoAllocChunkElems = int64_t(1) << 16;
constexpr int64_t kNoAllocMaxChunks = 16384;
constexpr int kMaxDevices = 64;

// Shared by every call on a device; each call overwrites the partials it reads.
static __device__ __align__(256) StatPartial g_noalloc_partials[kNoAllocMaxChunks];

template <int DT>
__global__ void __launch_bounds__(kBlock) noalloc_chunk_sums_kernel(const void* theta, const void* theta0,
                                                                    int64_t numel, uint32_t vec,
                                                                    StatPartial* partials) {
  __shared__ double sh_s[kBlock / 32];
  __shared__ double sh_q[kBlock / 32];
  DevTensor T;
  T.theta = theta;
  T.theta0 = theta0;
  T.flags = vec ? TF_VEC : 0u;
  const int64_t n_chunks = (numel + kNoAllocChunkElems - 1) / kNoAllocChunkElems;
  for (int64_t c = blockIdx.x; c < n_chunks; c += gridDim.x) {
    Chunk ch;
    ch.tensor = 0;
    ch.pad = 0;
    ch.begin = c * kNoAllocChunkElems;
    ch.end = (c + 1) * kNoAllocChunkElems < numel ? (c + 1) * kNoAllocChunkElems : numel;
    double ds, dq;
    chunk_delta_sums<DT>(T, ch, sh_s, sh_q, ds, dq);
    if (threadIdx.x == 0) {
      partials[c].sum = ds;
      partials[c].sumsq = dq;
    }
  }
}

// One CTA: sum the chunk partials in chunk order, then sigma.
__global__ void __launch_bounds__(kBlock) noalloc_sigma_kernel(const StatPartial* partials, int64_t n_chunks,
                                                               int64_t numel, float sigma_rel, float* out) {
  __shared__ double sh_s[kBlock / 32];
  __shared__ double sh_q[kBlock / 32];
  double s = 0.0, q = 0.0;
  for (int64_t k = threadIdx.x; k < n_chunks; k += kBlock) {
    s += partials[k].sum;
    q += partials[k].sumsq;
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
    *out = sigma_from_sums(ts, tq, numel, sigma_rel);
  }
}

smat_status record_error(smat_status s, const char* msg) {
  return (smat_status)record_error_code((int)s, msg);
}

std::mutex g_symbol_mutex;
StatPartial* g_symbol_ptr[kMaxDevices] = {};

}  // namespace
}  // namespace smat

using namespace smat;

extern "C" smat_status smat_delta_sigma_noalloc(const void* d_theta, const void* d_theta0, int64_t numel,
                                                int32_t dtype, float sigma_rel, float* d_sigma,
                                                smat_stream_t stream) {
  if (!d_sigma) return record_error(SMAT_ERR_INVALID_ARG, "d_sigma is NULL");
  if (dtype != SMAT_F32 && dtype != SMAT_BF16) return record_error(SMAT_ERR_UNSUPPORTED, "dtype not supported");
  if (numel < 0 || !(sigma_rel >= 0.0f) || sigma_rel > 3.0e38f)
    return record_error(SMAT_ERR_INVALID_ARG, "numel < 0 or sigma_rel invalid");
  const int64_t n_chunks = (numel + kNoAllocChunkElems - 1) / kNoAllocChunkElems;
  if (n_chunks > kNoAllocMaxChunks)
    return record_error(SMAT_ERR_INVALID_ARG,
                        "numel exceeds the fixed scratch array of the allocation-free entry point "
                        "(at most 16384 * 65536 = 1073741824 elements)");
  const size_t es = dtype == SMAT_BF16 ? 2 : 4;
  if (numel > 0) {
    if (!d_theta || !d_theta0) return record_error(SMAT_ERR_INVALID_ARG, "NULL data pointer");
    if ((uintptr_t)d_theta % es || (uintptr_t)d_theta0 % es)
      return record_error(SMAT_ERR_ALIGNMENT, "pointer not aligned to its element size");
  }
  if ((uintptr_t)d_sigma % 4) return record_error(SMAT_ERR_ALIGNMENT, "d_sigma not 4-byte aligned");

  // Set-up, once per device, with that device current: the array's device
  // address (its name in host code is only a host-side stand-in).
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return record_error(SMAT_ERR_CUDA, "no usable current device");
  StatPartial* partials = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_symbol_mutex);
    if (!g_symbol_ptr[dev]) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_noalloc_partials) != cudaSuccess || !p)
        return record_error(SMAT_ERR_CUDA, "cudaGetSymbolAddress of the scratch array failed");
      g_symbol_ptr[dev] = static_cast<StatPartial*>(p);
    }
    partials = g_symbol_ptr[dev];
  }

  if (n_chunks > 0) {
    int sms = 1;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return record_error(SMAT_ERR_CUDA, "device attribute query failed");
    const int64_t grid = n_chunks < 4 * (int64_t)sms ? n_chunks : 4 * (int64_t)sms;
    const uint32_t vec = ((uintptr_t)d_theta % 32 == 0 && (uintptr_t)d_theta0 % 32 == 0) ? 1u : 0u;
    if (dtype == SMAT_BF16)
      noalloc_chunk_sums_kernel<DT_BF16><<<(int)grid, kBlock, 0, stream>>>(d_theta, d_theta0, numel, vec, partials);
    else
      noalloc_chunk_sums_kernel<DT_F32><<<(int)grid, kBlock, 0, stream>>>(d_theta, d_theta0, numel, vec, partials);
    if (cudaGetLastError() != cudaSuccess) return record_error(SMAT_ERR_CUDA, "chunk sums launch failed");
  }
  noalloc_sigma_kernel<<<1, kBlock, 0, stream>>>(partials, n_chunks, numel, sigma_rel, d_sigma);
  if (cudaGetLastError() != cudaSuccess) return record_error(SMAT_ERR_CUDA, "sigma launch failed");
  return SMAT_OK;
}
